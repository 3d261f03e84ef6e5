// Tensor-core integer GEMMs for sm_103a (tcgen05 + TMEM + TMA).
//
// C[r, n] = sum_k A[r, k] B[n, k] with both operands K-major:
//   A: packed +-1 signs (uint32 words) or uint8 gradient codes,
//   B: packed +-1 signs.
// The binary product of App. C (XNOR-popcount) and the bit-plane product of
// Sec. 5.2 are evaluated exactly on the fp8 tensor cores: +-1 and codes
// 0..15 are exact e4m3 values, a b = 8 code is split into 16*hi + lo with
// both digits exact, products are exact, and every partial sum is an integer
// below 2^24 so the fp32 accumulator in TMEM holds it exactly.
//
// Pipeline per CTA (one 128 x BN output tile, 128-element K steps), two rings:
//   raw ring (deep)    TMA writes the raw tiles: packed sign words (16 bytes per row)
//                      or uint8 codes (128B-swizzled box)
//   operand ring       e4m3 A stages in TMEM (row = lane, 4 elements per column), e4m3 B
//                      tiles in shared memory in the 128B-swizzle K-major layout
//   warp 0 lane 0   TMA producer of the raw ring
//   warp 1          TMEM allocation; lane 0 issues tcgen05.mma (A from TMEM, B from shared
//                   memory) and commits operand stages
//   warps 2..5      expand A rows of their TMEM lane quarter and store them with tcgen05.st
//   warps 6..9      expand B rows into the shared tile
//   warps 2..9      then the epilogue: TMEM -> registers -> global memory (warp w owns TMEM
//                   lanes 32 (w % 4) .. +31 and half of the columns)
// Every wait is bounded; an expired wait sets FQT1_DEV_TIMEOUT and the CTA
// drains and returns.
#include <cuda.h>
#include <cudaTypedefs.h>

#include "gemm.cuh"

namespace fqt1 {

constexpr int kBM = 128;           // output rows per CTA (MMA M)
constexpr int kBK = 128;           // contraction elements per sub-tile (one 128-byte swizzle row of e4m3)
constexpr int kMaxStages = 8;
constexpr int kExpWarps = 8;       // two expansion / epilogue warps per SM sub-partition
constexpr int kThreads = 32 * (2 + kExpWarps);
constexpr uint64_t kWaitNs = 2000000000ull;  // 2 s bound on every wait
constexpr int kFoldTile = 128 * 129 * 4;  // Folder epilogue: int32 accumulator tile (aliases the rings)
constexpr int kFoldTab = 40960;           // Folder tables, a region of their own (bytes)
constexpr int kFoldZero = 4096;           // its last 4 KB: zeros, the source of bulk stores

enum : int { EPI_FWD = 0, EPI_ACC32 = 1, EPI_RED = 2, EPI_DX = 3, EPI_FOLD = 4, EPI_CRED = 5 };

struct TcArgs {
  int64_t M, N, L;           // rows (capacity), columns, contraction length
  const int32_t* count;      // valid rows = *count * rows_per_count (null: all M)
  int64_t rows_per_count;
  int k_tiles, tiles_per_split;
  int epi;
  const float* gamma;        // EPI_FWD: y = gamma[n] * acc (+ bias[n])
  const float* bias;         // EPI_FWD: per-column bias or null
  float* y;
  int32_t* acc;              // EPI_FWD (optional), EPI_ACC32, EPI_RED
  int64_t ldo;
  const int32_t* kept_idx;   // EPI_DX: dx[kept_idx[r / rpg] * rpg + r % rpg, n] = S' acc + Z' cs[n]
  const float* scale;
  const float* zero;
  const int32_t* cs;
  int64_t rpg;
  int32_t* status;
  // persistent tile loop (mode bit 7): output tiles p_tiles, p_tiles_n of them along N
  int64_t p_tiles, p_tiles_n;
  // EPI_FOLD: grad_input of a convolution with the Folder in the epilogue.  A CTA's rows are
  // whole samples (rpg = Ho*Wo divides 128) and its columns the kernel taps of fcb channels
  // starting at channel blockIdx.x * fcb (column offset n_step = fcb * kh * kw).
  int n_step, grid_x;
  int fC, fH, fW, fkh, fkw, fstride, fpad, fHo, fWo, fcb;
  // EPI_FWD / EPI_ACC32: bit 0 = y, bit 1 = acc leave through TMA stores (tmY / tmAcc)
  int tma_out;
  int fN;  // EPI_FOLD: samples (pruned ones are zeroed by the kernel; mode bit 2: dx in NHWC order)
  // implicit-GEMM forward of a stride-1 "same" convolution (mode bit 0): A comes from the
  // pixel-major sign words [N][H][W][C / 32] through a 4-D tensor map, one box per 128-channel
  // sub-tile of one kernel tap, shifted by the tap; the contraction index is k' = t C + c.
  // A box covers 2^isb consecutive sub-tiles of one tap (rows of 16 * 2^isb bytes).
  // (Mode bit 1: B is given as e4m3 bytes, +1 = 0x38, -1 = 0xB8, K-major rows, tmB a
  // 128B-swizzled map of 128 x 128 boxes, and goes by TMA straight into the operand ring; all
  // eight expansion warps then expand A, each half of a stage's sub-tiles.)
  int iC, ikw, ikhw, ipad, iW, iHW, isb;
  // EPI_FOLD divisors (host-built): kh kw, W, kw, H W, stride, fcb H W
  FastDiv fd_khw, fd_w, fd_kw, fd_hw, fd_s, fd_cbhw;
  // EPI_CRED: the cluster's partial tiles are summed into acc (int32, ldo) and dequantized into
  // y = dw[D][ldo] (kept channel kept_idx[r]: scale[r] acc + zero[r] cs[n]; pruned channels 0)
  const int32_t* slot_of_group;
  int64_t D;
  // EPI_ACC32: 1 = acc is column-major int32, acc[col * ldo + row]; a warp's 32 rows of one
  // column are then one 128-byte line, stored straight from the TMEM registers; 2 = the same
  // as int16 (the host checks that every sum fits: (2^b - 1) * contraction < 2^15)
  int acc_cm;
};

__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ uint64_t gtimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void mbar_init(uint64_t* b, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(b)), "r"(count));
}
__device__ __forceinline__ void mbar_arrive(uint64_t* b) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(b)) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* b, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(b)), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool mbar_test(uint64_t* b, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n.reg .pred p;\nmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\nselp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(smem_u32(b)), "r"(parity)
      : "memory");
  return ok != 0;
}
// Bounded wait for phase `parity` of barrier b; false (and the timeout status) if it expired
// or another role already gave up.
__device__ __forceinline__ bool mbar_wait(uint64_t* b, uint32_t parity, volatile int* abort_flag, int32_t* status,
                                          uint64_t limit_ns = kWaitNs) {
  if (mbar_test(b, parity)) return true;
  const uint64_t t0 = gtimer();
  for (uint32_t n = 1;; ++n) {
    if (mbar_test(b, parity)) return true;
    if ((n & 1023u) == 0) {  // the timer and the abort flag are checked every 1024 polls
      if (*abort_flag) return false;
      if (gtimer() - t0 > limit_ns) {
        *abort_flag = 1;
        if (status) atomicOr(status, FQT1_DEV_TIMEOUT);
        return false;
      }
    }
  }
}

__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, uint64_t* bar, int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], [%2];" ::"r"(
          smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(x), "r"(y)
      : "memory");
}

// 4-D tile load (coordinates innermost first; a box reaching outside the tensor reads zeros).
__device__ __forceinline__ void tma_load_4d(void* dst, const CUtensorMap* map, uint64_t* bar, int c0, int c1, int c2,
                                            int c3) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4, %5, %6}], "
      "[%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(c0), "r"(c1), "r"(c2), "r"(c3)
      : "memory");
}

// Shared -> global tile store through TMA (bulk group; the caller commits and waits).
__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, const void* src, int x, int y) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%2, %3}], [%1];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(smem_u32(src)), "r"(x), "r"(y)
               : "memory");
}

// Untiled bulk copy shared -> global (both addresses 16-byte aligned, bytes a multiple of 16).
__device__ __forceinline__ void bulk_store(void* gdst, const void* ssrc, uint32_t bytes) {
  asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(reinterpret_cast<uint64_t>(gdst)),
               "r"(smem_u32(ssrc)), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\nbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_size() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(r));
  return r;
}
// 16 bytes of CTA `rank`'s shared memory at this CTA's shared address saddr.
__device__ __forceinline__ int4 ld_cluster_v4(uint32_t saddr, uint32_t rank) {
  uint32_t ra;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(ra) : "r"(saddr), "r"(rank));
  int4 v;
  asm volatile("ld.shared::cluster.v4.s32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "r"(ra)
               : "memory");
  return v;
}
// Byte offset of 16-byte chunk ch (0..31) of row r (0..127) of a 128 x 128 int32 tile, the
// chunk index swizzled with r & 7 so that a warp's 32 rows hit distinct banks.
__device__ __forceinline__ uint32_t ptile_off(int r, int ch) { return (uint32_t)(r * 512 + ((ch ^ (r & 7)) << 4)); }

// Shared-memory matrix descriptor of a K-major operand tile in the 128-byte swizzle layout
// (rows of 128 bytes, 8-row groups 1024 bytes apart).
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFF) >> 4);
  d |= (uint64_t)1 << 16;              // leading byte offset (unused for this layout)
  d |= (uint64_t)(1024 >> 4) << 32;    // stride byte offset: next 8-row group
  d |= (uint64_t)1 << 46;              // descriptor version
  d |= (uint64_t)2 << 61;              // 128-byte swizzle
  return d;
}

// Instruction descriptor: e4m3 x e4m3 -> f32, both K-major, M = 128, N = bn.
__host__ __device__ constexpr uint32_t idesc_e4m3(int bn) {
  return (1u << 4) | (0u << 7) | (0u << 10) | ((uint32_t)(bn >> 3) << 17) | ((uint32_t)(kBM >> 4) << 24);
}

__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
               : "memory");
}

// A operand in TMEM (row = lane, 4 e4m3 per 32-bit column), B from a shared-memory descriptor.
__device__ __forceinline__ void mma_e4m3_ta(uint32_t tmem_d, uint32_t tmem_a, uint64_t bd, uint32_t idesc,
                                            uint32_t acc) {
  asm volatile(
      "{\n.reg .pred p;\nsetp.ne.b32 p, %4, 0;\n"
      "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], [%1], %2, %3, p;\n}\n" ::"r"(tmem_d),
      "r"(tmem_a), "l"(bd), "r"(idesc), "r"(acc));
}

// A and B both from shared-memory descriptors.
__device__ __forceinline__ void mma_e4m3_ss(uint32_t tmem_d, uint64_t ad, uint64_t bd, uint32_t idesc, uint32_t acc) {
  asm volatile(
      "{\n.reg .pred p;\nsetp.ne.b32 p, %4, 0;\n"
      "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n}\n" ::"r"(tmem_d),
      "l"(ad), "l"(bd), "r"(idesc), "r"(acc));
}

// An fp32 accumulator word -> the exact int32 sum.  With A_DIRECT the A operand was the code
// bytes themselves, read as e4m3: byte q < 16 is the e4m3 number q 2^-9 (subnormals 0..7,
// then the first binade 8..15), so the accumulator holds sum 2^-9 and 512 rescales it exactly.
// (A operands of e4m3 signs, +-1, need no rescale: A_DIRECT is false for them.)
template <bool A_DIRECT>
__device__ __forceinline__ int32_t acc_int(uint32_t v) {
  if constexpr (A_DIRECT) return __float2int_rn(__fmul_rn(__uint_as_float(v), 512.0f));
  else return __float2int_rn(__uint_as_float(v));
}

// 32 consecutive TMEM columns of this thread's lane <- v (the warp writes its 32 lanes).
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&v)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,"
      "%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
      "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]),
      "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15]), "r"(v[16]), "r"(v[17]),
      "r"(v[18]), "r"(v[19]), "r"(v[20]), "r"(v[21]), "r"(v[22]), "r"(v[23]), "r"(v[24]), "r"(v[25]), "r"(v[26]),
      "r"(v[27]), "r"(v[28]), "r"(v[29]), "r"(v[30]), "r"(v[31])
      : "memory");
}

// Folder of a 3 x 3, stride-1, pad-1 convolution (Ho = H, Wo = W): tap offsets are computed,
// not looked up.
__device__ __forceinline__ bool fold_same3(const TcArgs& a) {
  return a.fkh == 3 && a.fkw == 3 && a.fstride == 1 && a.fpad == 1;
}

// Sub-tiles of stage kt that hold contraction elements below L (1..KSUB for a stage that
// starts below L).
template <int KSUB>
__device__ __forceinline__ int valid_subtiles(int64_t L, int kt) {
  const int64_t left = L - (int64_t)kt * KSUB * kBK;
  return left >= (int64_t)KSUB * kBK ? KSUB : (int)((left + kBK - 1) / kBK);
}

// Byte offset of 16-byte chunk c of row r in a 128B-swizzled tile.
__device__ __forceinline__ uint32_t swz(int r, int c) {
  return (uint32_t)((r >> 3) * 1024 + (r & 7) * 128 + ((c ^ (r & 7)) << 4));
}

// 4 sign bits (bits 0..3 of nib) -> 4 e4m3 bytes (+1 = 0x38, -1 = 0xB8).  The product holds
// four copies of nib shifted by 7, 14, 21 and 28 bits; they do not overlap, and bit k of the
// copy shifted by 7 (k + 1) lands on bit 8k + 7, the sign bit of byte k.
__device__ __forceinline__ uint32_t signs4(uint32_t nib) {
  return ((nib * 0x10204080u) & 0x80808080u) ^ 0xB8B8B8B8u;
}
// 16 sign bits -> 16 e4m3 bytes.
__device__ __forceinline__ uint4 signs16(uint32_t h) {
  return make_uint4(signs4(h & 15u), signs4((h >> 4) & 15u), signs4((h >> 8) & 15u), signs4((h >> 12) & 15u));
}
// 4 codes (one per byte, each < 16) -> 4 e4m3 bytes of the same integers.
__device__ __forceinline__ uint32_t codes4(uint32_t c) {
  const uint32_t y = c & 0x07070707u;
  // low 3 bits of byte i -> selector nibble i (bytes 0 and 2 of y | y >> 4 hold two nibbles each)
  const uint32_t sel = __byte_perm(y | (y >> 4), 0u, 0x0020u);
  const uint32_t lo = __byte_perm(0x44403800u, 0x4E4C4A48u, sel);  // e4m3 of 0..7
  const uint32_t hi = __byte_perm(0x53525150u, 0x57565554u, sel);  // e4m3 of 8..15
  // 0xFF in the bytes whose code is >= 8: bit 3 moved to the byte's sign bit, then replicated
  // over the byte by prmt.b32 (a selector nibble with its top bit set sign-extends the byte;
  // __byte_perm ignores that bit, hence the inline PTX)
  uint32_t m;
  asm("prmt.b32 %0, %1, %2, %3;" : "=r"(m) : "r"(c << 4), "r"(0u), "r"(0xBA98u));
  return (lo & ~m) | (hi & m);
}
// e4m3 of 16*h for digits h < 16 (exponent raised by 4; zero stays zero).
__device__ __forceinline__ uint32_t codes4_x16(uint32_t h) {
  const uint32_t e = codes4(h);
  // every nonzero byte of e is in 0x38..0x57, so adding 0x7F sets its top bit without a carry
  const uint32_t nz = ((e + 0x7F7F7F7Fu) & 0x80808080u) >> 2;  // 0x20 per nonzero byte
  return e + nz;
}

// TAB: SHORT tiles of the fused Folder keep its tables after the rings; other SHORT tiles do not.
template <bool A_CODES, bool BITS8, int BN, bool SHORT = false, bool TAB = SHORT>
struct TcSmem {
  static_assert(BN == 128, "one B row per expansion thread");
  // a stage carries KSUB sub-tiles of kBK contraction elements (fewer ring hand-offs per element)
  static constexpr int KSUB = A_CODES ? 2 : 4;
  static constexpr int kSub = BN * kBK;                          // bytes of one e4m3 B sub-tile
  static constexpr int kOpB = kSub * KSUB;                        // bytes of one B stage (shared)
  static constexpr int kAcols = (kBK / 4) * KSUB * (BITS8 ? 2 : 1);  // TMEM columns of one A stage
  static constexpr int kRawRow = 16 * KSUB;                       // packed-sign bytes per row per stage
  static constexpr int kRawA = A_CODES ? kBM * kBK * KSUB : kBM * kRawRow;
  static constexpr int kRawB = BN * kRawRow;
  static constexpr int kRawStage = kRawA + kRawB;
  // SHORT: single-buffered rings for short contractions (two CTAs per SM)
  static constexpr int kOpStages = SHORT ? 1 : 2;
  static constexpr int kRawStages = SHORT ? 1 : (A_CODES ? 3 : 4);
  // TMEM: the BN accumulator columns, then the A stages
  static constexpr int kTmemUsed = BN + kOpStages * kAcols;
  static constexpr int kTmemCols = kTmemUsed <= 256 ? 256 : 512;
  static constexpr int kRing = kOpStages * kOpB + kRawStages * kRawStage;
  // the epilogue reuses the rings (per-warp staging, or the Folder's accumulator tile); the
  // Folder's tables have a region of their own after the rings (built while the rings are busy)
  static constexpr int kEpi = SHORT ? kFoldTile : kExpWarps * 16384;
  static constexpr int kMain = kRing > kEpi ? kRing : kEpi;
  static constexpr int kTab = SHORT && TAB ? kFoldTab : 0;
  static constexpr int kBytes = kMain + kTab + 1024;  // + alignment slack
  static_assert(kSub % 1024 == 0 && kRawStage % 1024 == 0, "stages keep 1024-byte alignment");
  static_assert(kTmemUsed <= 512, "TMEM holds 512 columns");
  static_assert(!SHORT || kTmemCols <= 256, "two CTAs per SM share the TMEM columns");
  static_assert(kBytes <= 227 * 1024, "shared memory per CTA");
  static_assert(!A_CODES || kBK * KSUB == kCodesStageK, "the host sizes code stages with kCodesStageK");
};

// SHORT tiles run two CTAs per SM, which caps the registers at 65536 / (2 * 320) per thread.
// X selects the optional datapaths at compile time, so that the default kernels carry none of
// their code: bit 0 the implicit-convolution A operand, bit 1 B as e4m3 bytes by TMA (b_tma),
// bit 2 the Folder's NHWC output, bit 3 codes of at most 4 bits as the A operand straight from
// the raw ring (A_DIRECT: the MMA reads the TMA-written code tile as e4m3, nothing expands A;
// the raw stage is released by the MMA's commit), bit 4 the failure-path test: the expansion
// warps withhold their arrive on the first operand stage, so the MMA issuer's bounded wait
// (20 ms in this instantiation) expires and the kernel takes its timeout exit, bit 6 a SHORT
// tile without the Folder's tables (two CTAs per SM for short contractions; a TMA-stored
// output is y alone), bit 5 e4m3
// signs (+1 = 0x38, -1 = 0xB8) as the A operand straight from the raw ring (the A_DIRECT
// datapath with a unit scale: the forward product of e4m3 X_u rows).
template <bool A_CODES, bool BITS8, int BN, bool SHORT, int X = 0>
__global__ void __launch_bounds__(kThreads, SHORT ? 2 : 1)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ CUtensorMap tmY, const __grid_constant__ CUtensorMap tmAcc, TcArgs a) {
  using S = TcSmem<A_CODES, BITS8, BN, SHORT, (X & 64) == 0>;
  constexpr bool kImpl = (X & 1) != 0, kBtma = (X & 2) != 0, kNhwc = (X & 4) != 0;
  // bit 3: codes below 16 as the A operand straight from TMA (scale 2^-9); bit 5: e4m3 signs
  // (+-1) as the A operand straight from TMA (scale 1).  Both take the A_DIRECT datapath.
  constexpr bool kA512 = (X & 8) != 0, kAdir = (X & 8) != 0 || (X & 32) != 0;
  static_assert(!kAdir || (A_CODES && !BITS8), "A_DIRECT takes byte operands of one digit");
  constexpr bool kLose = (X & 16) != 0;
  // bit 7: a persistent CTA takes output tiles blockIdx.x, + gridDim.x, ... (EPI_FWD / EPI_ACC32 /
  // EPI_DX without splits): the set-up is paid once, the producer loads the next tile's stages
  // while the epilogue of the current one runs, and the rings' positions and phases continue
  // across tiles
  constexpr bool kPersist = (X & 128) != 0;
  constexpr uint64_t kLimit = kLose ? 20000000ull : kWaitNs;  // bound of every wait below
  // arrivals that free a raw stage: the expansion warps (when they read it) and, with A_DIRECT,
  // the commit of the MMAs that read its A tile
  constexpr uint32_t kRawEmpty = kAdir ? (kBtma ? 1u : (uint32_t)kExpWarps + 1u) : (uint32_t)kExpWarps;
  constexpr int OS = S::kOpStages, RS = S::kRawStages, KSUB = S::KSUB;
  extern __shared__ unsigned char smem_raw[];
  __shared__ __align__(8) uint64_t raw_full[kMaxStages], raw_empty[kMaxStages], op_full[kMaxStages],
      op_empty[kMaxStages];
  __shared__ __align__(8) uint64_t acc_full;
  __shared__ __align__(8) uint64_t b_full[kMaxStages];  // b_tma: the B boxes of an operand stage landed
  __shared__ uint32_t tmem_slot;
  __shared__ volatile int abort_flag;
  __shared__ __align__(16) float gamma_s[BN];  // EPI_FWD: Gamma of this tile's columns (read as float4)
  __shared__ __align__(16) float bias_s[BN];   // EPI_FWD with a bias: the bias of those columns

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int64_t m0 = (int64_t)blockIdx.y * kBM, n0 = (int64_t)blockIdx.x * (a.n_step > 0 ? a.n_step : BN);
  const int kt0 = blockIdx.z * a.tiles_per_split;
  const int kt1 = min(a.k_tiles, kt0 + a.tiles_per_split);
  if (kt0 >= kt1) {
    FQT1_PDL_TRIGGER();
    return;
  }

  // 1024-byte aligned start of the dynamic shared memory, derived from smem_raw by an offset
  // (not by a round trip through an integer) so that accesses through it stay shared-memory
  // accesses instead of generic ones
  unsigned char* base = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  auto opB = [&](int s) { return base + s * S::kOpB; };
  unsigned char* raw_base = base + OS * S::kOpB;
  auto rawA = [&](int s) { return raw_base + s * S::kRawStage; };
  auto rawB = [&](int s) { return raw_base + s * S::kRawStage + S::kRawA; };

  if (threadIdx.x == 0) {
    abort_flag = 0;
    for (int s = 0; s < RS; ++s) { mbar_init(&raw_full[s], 1); mbar_init(&raw_empty[s], kRawEmpty); }
    for (int s = 0; s < OS; ++s) { mbar_init(&op_full[s], kExpWarps); mbar_init(&op_empty[s], 1); mbar_init(&b_full[s], 1); }
    mbar_init(&acc_full, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tmem_slot)),
                 "r"(S::kTmemCols));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  if (threadIdx.x == 0) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmA)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmB)) : "memory");
  }
  // Folder tap table (geometry only, so it is built before the dependency wait): for input
  // position pos = h W + w and tap t = i kw + j, the accumulator tile offset
  // (output pixel * 129 + t) of the product that lands there, or -1
  int32_t* const fold_tab = reinterpret_cast<int32_t*>(base + S::kMain);
  if (SHORT && a.epi == EPI_FOLD && threadIdx.x >= 64) {
    int4* zb = reinterpret_cast<int4*>(base + S::kMain + kFoldTab - kFoldZero);
    for (int x = threadIdx.x - 64; x < kFoldZero / 16; x += 256) zb[x] = make_int4(0, 0, 0, 0);
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // the bulk stores read it later
  }
  if (SHORT && a.epi == EPI_FOLD && threadIdx.x >= 64 && !fold_same3(a)) {  // same 3x3: offsets computed
    const int khw = a.fkh * a.fkw, HW = a.fH * a.fW;
    for (int x = threadIdx.x - 64; x < HW * khw; x += 256) {
      const int pos = (int)a.fd_khw.div((uint32_t)x), t = x - pos * khw;
      const int h = (int)a.fd_w.div((uint32_t)pos), w = pos - h * a.fW;
      const int i = (int)a.fd_kw.div((uint32_t)t), j = t - i * a.fkw;
      const int hn = h + a.fpad - i, wn = w + a.fpad - j;
      int v = -1;
      if (hn >= 0 && wn >= 0) {
        const int oh = (int)a.fd_s.div((uint32_t)hn), ow = (int)a.fd_s.div((uint32_t)wn);
        if (oh * a.fstride == hn && ow * a.fstride == wn && oh < a.fHo && ow < a.fWo)
          v = (oh * a.fWo + ow) * (BN + 1) + t;
      }
      fold_tab[x] = v;
    }
  }
  // lane 0 of warp 0 ran alone above; __syncthreads is an aligned barrier (all lanes of a
  // warp must reach it together), so reconverge first
  __syncwarp();
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = tmem_slot;
  // the setup above overlaps the previous kernel; operands and the kept count are read after this
  FQT1_PDL_WAIT();
  FQT1_PDL_TRIGGER();
  const int64_t valid_rows = a.count ? (int64_t)__ldg(a.count) * a.rows_per_count : a.M;

  const uint32_t kTx = kBtma ? (uint32_t)S::kRawA : (uint32_t)S::kRawStage;
  int gbase = 0;     // operand stages of this CTA's earlier tiles
  int issued = 0;    // producer: raw stages issued
  int b_issued = 0;  // b_tma: operand stages whose B boxes this thread (warp 2, lane 0) issued
  const int64_t ptiles = kPersist ? a.p_tiles : 1;
  for (int64_t pt = kPersist ? (int64_t)blockIdx.x : 0, tj = 0; pt < ptiles; pt += kPersist ? gridDim.x : 1, ++tj) {
  if (kPersist) {
    m0 = (pt / a.p_tiles_n) * kBM;
    n0 = (pt % a.p_tiles_n) * BN;
  }
  const int nk = m0 < valid_rows ? kt1 - kt0 : 0;  // a tile past the kept rows has no work

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer (raw ring)
    if (lane == 0) {
      for (int i = 0; i < nk; ++i) {
        const int g = gbase + i, s = g % RS, it = g / RS;
        if (it > 0 && !mbar_wait(&raw_empty[s], (it - 1) & 1, &abort_flag, a.status, kLimit)) break;
        const int kt = kt0 + i;
        mbar_expect_tx(&raw_full[s], kTx);
        if (A_CODES) {
#pragma unroll
          for (int h = 0; h < KSUB; ++h)  // one 128-byte-swizzled box per sub-tile
            tma_load_2d(rawA(s) + h * (kBM * kBK), &tmA, &raw_full[s], (kt * KSUB + h) * kBK, (int)m0);
        } else if (!A_CODES && kImpl) {
          // implicit convolution: box b = sub-tiles b 2^isb .. + 2^isb - 1, 128 2^isb channels
          // of one tap t; the box of the tile's output pixels shifted by (i - pad, j - pad), so
          // that a tap in the padding reads the fill value 0 (sign -1).  Boxes past the
          // contraction length load a valid box whose products are never issued.
          const int64_t pix_n0 = m0 / a.iHW, pix_h0 = (m0 - pix_n0 * a.iHW) / a.iW;
          const int sb = 1 << a.isb;
          for (int h = 0; h < KSUB; h += sb) {
            const int64_t kq = ((int64_t)kt * KSUB + h) * kBK;
            const int t = kq < a.L ? (int)(kq / a.iC) : a.ikhw - 1;
            const int cw = kq < a.L ? (int)((kq - (int64_t)t * a.iC) >> 5) : 0;
            const int ti = t / a.ikw, tj = t - ti * a.ikw;
            tma_load_4d(rawA(s) + h * (kBM * 16), &tmA, &raw_full[s], cw, tj - a.ipad,
                        (int)pix_h0 + ti - a.ipad, (int)pix_n0);
          }
        } else {
          tma_load_2d(rawA(s), &tmA, &raw_full[s], kt * KSUB * (kBK / 32), (int)m0);
        }
        if (!kBtma) tma_load_2d(rawB(s), &tmB, &raw_full[s], kt * KSUB * (kBK / 32), (int)n0);
        ++issued;
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer (operand ring)
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_e4m3(BN);
      for (int i = 0; i < nk; ++i) {
        const int g = gbase + i, s = g % OS, it = g / OS, sr = g % RS, itr = g / RS;
        if (!mbar_wait(&op_full[s], it & 1, &abort_flag, a.status, kLimit)) break;
        if (kBtma && !mbar_wait(&b_full[s], it & 1, &abort_flag, a.status, kLimit)) break;
        if (kAdir && !mbar_wait(&raw_full[sr], itr & 1, &abort_flag, a.status, kLimit)) break;  // the A codes landed
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const uint32_t acol = tmem + BN + s * S::kAcols, baddr = smem_u32(opB(s));
        const uint32_t aaddr = smem_u32(rawA(sr));
        const int nsub = valid_subtiles<KSUB>(a.L, kt0 + i);
#pragma unroll
        for (int h = 0; h < KSUB; ++h) {
          if (h >= nsub) break;  // sub-tiles past the contraction length hold no products
#pragma unroll
          for (int k = 0; k < kBK / 32; ++k) {
            const uint64_t bd = sw128_desc(baddr + h * S::kSub + 32 * k);
            const uint32_t first = (i > 0 || h > 0 || k > 0) ? 1u : 0u;
            if (kAdir) {
              mma_e4m3_ss(tmem, sw128_desc(aaddr + h * (kBM * kBK) + 32 * k), bd, idesc, first);
            } else {
              mma_e4m3_ta(tmem, acol + (kBK / 4) * h + 8 * k, bd, idesc, first);
              if (BITS8) mma_e4m3_ta(tmem, acol + (kBK / 4) * (KSUB + h) + 8 * k, bd, idesc, 1u);
            }
          }
        }
        mma_commit(&op_empty[s]);
        if (kAdir) mma_commit(&raw_empty[sr]);  // the A tile is free once these MMAs are done
      }
      mma_commit(&acc_full);
    }
  } else {
    // ---------------------------------------------------------------- expansion (raw -> operands)
    // warps 2..5: the 32 A rows of their TMEM lane quarter -> e4m3 in TMEM (one row per thread);
    // warps 6..9: B row 32 (warp - 6) + lane -> e4m3 in the 128B-swizzled shared tile
    // (the split below changes this for tiles with few live rows)
    // A tile with at most two live lane quarters (e.g. 64 kept channels) and two sub-tiles per
    // stage splits its A work by sub-tile over the two warps of each live quarter (4 / 8 and
    // 5 / 9); warps 2, 3, 6 and 7 then take the B rows.
    const int64_t tile_rows = valid_rows - m0;  // may exceed kBM or be negative
    const int live_q = tile_rows >= kBM ? 4 : (tile_rows <= 0 ? 0 : (int)((tile_rows + 31) / 32));
    // A_DIRECT: no A expansion; all eight warps expand B (or, with b_tma, nothing), warps 2..5
    // the first half of a stage's sub-tiles and warps 6..9 the second half, each warp the 32 B
    // rows of its lane quarter
    const bool split = !kAdir && KSUB == 2 && live_q <= 2;
    const bool a_warp = kAdir ? false : kBtma ? true : split ? (warp == 4 || warp == 5 || warp >= 8) : warp < 6;
    const int a_h0 = kBtma ? (warp >= 6 ? KSUB / 2 : 0) : (split && warp >= 8 ? 1 : 0);
    const int a_h1 = kBtma ? a_h0 + KSUB / 2 : (split ? a_h0 + 1 : KSUB);
    const int bblk = kAdir ? (warp & 3) : split ? (warp == 2 ? 0 : warp == 3 ? 1 : warp == 6 ? 2 : 3) : warp - 6;
    const int b_h0 = kAdir ? (warp >= 6 ? KSUB / 2 : 0) : 0, b_h1 = kAdir ? b_h0 + KSUB / 2 : KSUB;
    const int quarter = warp & 3;
    const int arow = 32 * quarter + lane, brow = 32 * bblk + lane;
    // a warp whose 32 A rows all lie past the kept rows skips its work: an accumulator row
    // depends only on its own A row, and the epilogue drops those rows
    const bool a_live = a_warp && m0 + 32 * quarter < valid_rows;
    const uint32_t a_lanes = tmem + ((uint32_t)(32 * quarter) << 16);
    for (int i = 0; i < nk; ++i) {
      const int g = gbase + i, so = g % OS, ito = g / OS, sr = g % RS, itr = g / RS;
      if (ito > 0 && !mbar_wait(&op_empty[so], (ito - 1) & 1, &abort_flag, a.status, kLimit)) break;
      if (kBtma) {  // the stage's B boxes, as soon as the MMAs of its previous use are done
        if (warp == 2 && lane == 0) {
          mbar_expect_tx(&b_full[so], (uint32_t)S::kOpB);
#pragma unroll
          for (int h = 0; h < KSUB; ++h)
            tma_load_2d(opB(so) + h * S::kSub, &tmB, &b_full[so], ((kt0 + i) * KSUB + h) * kBK, (int)n0);
          ++b_issued;
        }
        __syncwarp();
      }
      // with A_DIRECT and b_tma the expansion warps read nothing from the raw stage
      if (!(kAdir && kBtma) && !mbar_wait(&raw_full[sr], itr & 1, &abort_flag, a.status, kLimit)) break;
      const int kt = kt0 + i;
      if (kAdir && kBtma) {
        // nothing to expand: the arrive below only hands the B stage's issue to the MMA
      } else if (a_warp) {
        if (a_live) {
          const uint32_t acol = a_lanes + BN + so * S::kAcols;
          const int nsub = min(valid_subtiles<KSUB>(a.L, kt), a_h1);
#pragma unroll 1
          for (int h = a_h0; h < nsub; ++h) {  // one sub-tile's registers live at a time
            uint32_t o[32];
            if (A_CODES) {
              const unsigned char* ra = rawA(sr) + h * (kBM * kBK);
              if (BITS8) {
                uint32_t o2[32];
#pragma unroll
                for (int c = 0; c < 8; ++c) {  // TMA wrote the codes with the 128B swizzle
                  const uint4 v = *reinterpret_cast<const uint4*>(ra + swz(arow, c));
                  o[4 * c + 0] = codes4_x16((v.x >> 4) & 0x0F0F0F0Fu); o2[4 * c + 0] = codes4(v.x & 0x0F0F0F0Fu);
                  o[4 * c + 1] = codes4_x16((v.y >> 4) & 0x0F0F0F0Fu); o2[4 * c + 1] = codes4(v.y & 0x0F0F0F0Fu);
                  o[4 * c + 2] = codes4_x16((v.z >> 4) & 0x0F0F0F0Fu); o2[4 * c + 2] = codes4(v.z & 0x0F0F0F0Fu);
                  o[4 * c + 3] = codes4_x16((v.w >> 4) & 0x0F0F0F0Fu); o2[4 * c + 3] = codes4(v.w & 0x0F0F0F0Fu);
                }
                tmem_st32(acol + (kBK / 4) * h, o);
                tmem_st32(acol + (kBK / 4) * (KSUB + h), o2);
              } else {
#pragma unroll
                for (int c = 0; c < 8; ++c) {
                  const uint4 v = *reinterpret_cast<const uint4*>(ra + swz(arow, c));
                  o[4 * c + 0] = codes4(v.x); o[4 * c + 1] = codes4(v.y);
                  o[4 * c + 2] = codes4(v.z); o[4 * c + 3] = codes4(v.w);
                }
                tmem_st32(acol + (kBK / 4) * h, o);
              }
            } else {
              // raw rows: 16 bytes per sub-tile, interleaved per row (2-D box), or per row of a
              // box of 2^isb sub-tiles (implicit convolution)
              const int hb = (h >> a.isb) << a.isb;
              const unsigned char* rp = kImpl ? rawA(sr) + hb * (kBM * 16) + (arow << (4 + a.isb)) + 16 * (h - hb)
                                               : rawA(sr) + arow * S::kRawRow + 16 * h;
              const uint4 w4 = *reinterpret_cast<const uint4*>(rp);
              const uint32_t wv[4] = {w4.x, w4.y, w4.z, w4.w};
#pragma unroll
              for (int j = 0; j < 32; ++j) o[j] = signs4((wv[j >> 3] >> (4 * (j & 7))) & 15u);
              const int64_t kbase = ((int64_t)kt * KSUB + h) * kBK;
              if (kbase + kBK > a.L) {  // elements past the contraction length contribute 0
#pragma unroll
                for (int j = 0; j < 32; ++j) {
#pragma unroll
                  for (int bb = 0; bb < 4; ++bb)
                    if (kbase + 4 * j + bb >= a.L) o[j] &= ~(0xFFu << (8 * bb));
                }
              }
              tmem_st32(acol + (kBK / 4) * h, o);
            }
          }
          asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
        }
        asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
      } else {
        const int nsub = min(valid_subtiles<KSUB>(a.L, kt), b_h1);
#pragma unroll
        for (int h = b_h0; h < KSUB; ++h) {
          if (h >= nsub) break;
          const uint4 w4 = *reinterpret_cast<const uint4*>(rawB(sr) + brow * S::kRawRow + 16 * h);
          const uint32_t wv[4] = {w4.x, w4.y, w4.z, w4.w};
          unsigned char* tb = opB(so) + h * S::kSub;
#pragma unroll
          for (int w = 0; w < 4; ++w) {
            *reinterpret_cast<uint4*>(tb + swz(brow, 2 * w)) = signs16(wv[w]);
            *reinterpret_cast<uint4*>(tb + swz(brow, 2 * w + 1)) = signs16(wv[w] >> 16);
          }
        }
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      }
      __syncwarp();
      if (lane == 0) {
        if (!(kLose && i == 0)) mbar_arrive(&op_full[so]);
        if (!(kAdir && kBtma)) mbar_arrive(&raw_empty[sr]);
      }
    }

    // every B box this thread issued must land before the epilogue reuses the ring or the CTA
    // exits (normally the MMA issuer has already seen them land)
    if (kBtma && warp == 2 && lane == 0) {
      for (int i = (b_issued > OS ? b_issued - OS : 0); i < b_issued; ++i) {
        const int so = i % OS, ito = i / OS;
        const uint64_t t0 = gtimer();
        while (!mbar_test(&b_full[so], ito & 1) && gtimer() - t0 < kWaitNs) {
        }
      }
    }
    __syncwarp();

    // ---------------------------------------------------------------- epilogue
    // TMEM -> registers (thread = row) -> per-warp swizzled staging (32 x 32 words) ->
    // one coalesced 128-byte row per store instruction (lane = column).
    // Folder tables that read inputs (after the dependency wait, before the accumulator is
    // ready): this block's colsums, the folded colsum of each (channel, position), and each
    // sample's kept id, scale and zero point
    const int f_khw = a.fkh * a.fkw, f_HW = a.fH * a.fW, f_imgs = a.rpg > 0 ? kBM / (int)a.rpg : 0;
    const int f_c0 = blockIdx.x * a.fcb, f_nc = min(a.fcb, a.fC - f_c0);
    int32_t* const f_tap = fold_tab;                   // [HW][khw]
    int32_t* const f_csf = f_tap + f_HW * f_khw;       // [nc][HW]
    int32_t* const f_cs = f_csf + f_nc * f_HW;         // [nc * khw]
    float* const f_scale = reinterpret_cast<float*>(f_cs + f_nc * f_khw);
    float* const f_zero = f_scale + f_imgs;
    int32_t* const f_n = reinterpret_cast<int32_t*>(f_zero + f_imgs);
    bool fold_zero_issued = false;  // bulk stores of zeros in flight (read from shared memory)
    if (SHORT && a.epi == EPI_FOLD) {
      const int tt = threadIdx.x - 64;
      // every global load of the tables (column sums, kept count, kept ids, scales, zero
      // points, and the kept flags of this thread's first zeroing pieces below) is issued
      // together from clamped indices; the results are selected afterwards
      const int ncs = f_nc * f_khw;  // <= 128
      const int32_t cs_v = __ldg(a.cs + (int64_t)f_c0 * f_khw + min(tt, ncs - 1));
      const int64_t slot0 = (int64_t)blockIdx.y * f_imgs, cap = a.M / a.rpg;  // rpg divides 128
      const int64_t slot = min(slot0 + min(tt, f_imgs - 1), cap - 1);
      const int64_t nslots = __ldg(a.count);
      const int32_t kid = __ldg(a.kept_idx + slot);
      const float ksc = __ldg(a.scale + slot), kze = __ldg(a.zero + slot);
      const int nsamp = a.fN > (int)blockIdx.y ? (a.fN - (int)blockIdx.y + (int)gridDim.y - 1) / (int)gridDim.y : 0;
      // zeroing of a pruned sample: NCHW, this CTA's channel block (nc H W contiguous floats);
      // NHWC, the whole sample (C H W contiguous floats), its 4 KB pieces dealt round-robin over
      // the gridDim.x CTAs of the sample's row tile
      const int64_t blk_bytes = kNhwc ? (int64_t)a.fC * f_HW * 4 : (int64_t)f_nc * f_HW * 4;
      const int pieces_all = (int)((blk_bytes + kFoldZero - 1) / kFoldZero);
      const int pieces = !kNhwc ? pieces_all
                         : (pieces_all > (int)blockIdx.x
                                ? (pieces_all - (int)blockIdx.x + (int)gridDim.x - 1) / (int)gridDim.x : 0);
      int32_t sl[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int k = nsamp > 0 ? min(tt + 256 * u, nsamp * pieces - 1) / pieces : 0;
        sl[u] = __ldg(a.slot_of_group + min((int64_t)blockIdx.y + (int64_t)k * gridDim.y, (int64_t)a.fN - 1));
      }
      if (tt < ncs) f_cs[tt] = cs_v;
      if (tt < f_imgs) {
        const bool kept = slot0 + tt < nslots;
        f_n[tt] = kept ? kid : -1;
        f_scale[tt] = kept ? ksc : 0.f;
        f_zero[tt] = kept ? kze : 0.f;
      }
      asm volatile("bar.sync 1, 256;" ::: "memory");  // the 256 epilogue threads
      if (fold_same3(a) && 256 % f_HW == 0) {
        // one input position per thread (H W divides 256): its 9-tap validity mask once
        const int pos = tt & (f_HW - 1);
        const int h = (int)a.fd_w.div((uint32_t)pos), w = pos - h * a.fW;
        uint32_t msk = 0;
#pragma unroll
        for (int t = 0; t < 9; ++t)
          if ((unsigned)(h + 1 - t / 3) < (unsigned)a.fH && (unsigned)(w + 1 - t % 3) < (unsigned)a.fW) msk |= 1u << t;
        for (int cl = tt / f_HW; cl < f_nc; cl += 256 / f_HW) {
          int32_t cs = 0;
#pragma unroll
          for (int t = 0; t < 9; ++t) cs += (msk >> t) & 1u ? f_cs[cl * 9 + t] : 0;
          f_csf[cl * f_HW + pos] = cs;
        }
      }
      for (int x = tt; !(fold_same3(a) && 256 % f_HW == 0) && x < f_nc * f_HW; x += 256) {
        const int cl = (int)a.fd_hw.div((uint32_t)x), pos = x - cl * f_HW;
        int32_t cs = 0;
        if (fold_same3(a)) {  // tap (i, j) of input (h, w) lands on output (h + 1 - i, w + 1 - j)
          const int h = (int)a.fd_w.div((uint32_t)pos), w = pos - h * a.fW;
#pragma unroll
          for (int t = 0; t < 9; ++t)
            if ((unsigned)(h + 1 - t / 3) < (unsigned)a.fH && (unsigned)(w + 1 - t % 3) < (unsigned)a.fW)
              cs += f_cs[cl * 9 + t];
        } else {
          for (int t = 0; t < f_khw; ++t)
            if (f_tap[pos * f_khw + t] >= 0) cs += f_cs[cl * f_khw + t];
        }
        f_csf[x] = cs;
      }
      // pruned samples (they do not depend on the products, so before the accumulator is
      // ready): this CTA zeroes its channel block (nc HW contiguous floats) of samples
      // blockIdx.y, + gridDim.y, ...: bulk stores from a zero buffer, one thread per 4 KB piece;
      // the kept flags of a thread's pieces are loaded together first
      if (f_HW % 4 == 0) {
        const unsigned char* zb = base + S::kMain + kFoldTab - kFoldZero;
        for (int e0 = tt; e0 < nsamp * pieces; e0 += 4 * 256) {
          if (e0 != tt) {  // later pieces (the first ones' flags were loaded with the tables)
#pragma unroll
            for (int u = 0; u < 4; ++u) {
              const int k = min(e0 + 256 * u, nsamp * pieces - 1) / pieces;
              sl[u] = __ldg(a.slot_of_group + (int64_t)blockIdx.y + (int64_t)k * gridDim.y);
            }
          }
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int e = e0 + 256 * u;
            if (e >= nsamp * pieces || sl[u] >= 0) continue;
            const int k = e / pieces, pj = e - k * pieces;
            const int pc = kNhwc ? (int)blockIdx.x + pj * (int)gridDim.x : pj;
            const int64_t n = (int64_t)blockIdx.y + (int64_t)k * gridDim.y;
            const int64_t first = kNhwc ? (int64_t)n * a.fC * f_HW : ((int64_t)n * a.fC + f_c0) * f_HW;
            unsigned char* dst = reinterpret_cast<unsigned char*>(a.y + first) + (int64_t)pc * kFoldZero;
            const int64_t left = blk_bytes - (int64_t)pc * kFoldZero;
            bulk_store(dst, zb, (uint32_t)(left < kFoldZero ? left : kFoldZero));
            fold_zero_issued = true;
          }
        }
        if (fold_zero_issued) asm volatile("cp.async.bulk.commit_group;" ::: "memory");
      } else {
        const int per_img = a.fcb * f_HW;
        for (int e = tt; e < nsamp * per_img; e += 256) {
          const int k = (int)a.fd_cbhw.div((uint32_t)e), x = e - k * per_img;
          if (x >= f_nc * f_HW) continue;
          const int64_t n = (int64_t)blockIdx.y + (int64_t)k * gridDim.y;
          if (__ldg(a.slot_of_group + n) >= 0) continue;
          a.y[((int64_t)n * a.fC + f_c0) * f_HW + x] = 0.f;
        }
      }
    }
    if (a.tma_out & 1) {  // Gamma of this tile's columns, before the accumulator is ready
      const int tt = threadIdx.x - 64;
      if (tt < BN) gamma_s[tt] = n0 + tt < a.N ? __ldg(a.gamma + n0 + tt) : 0.f;
      if (a.bias && tt < BN) bias_s[tt] = n0 + tt < a.N ? __ldg(a.bias + n0 + tt) : 0.f;
      asm volatile("bar.sync 1, 256;" ::: "memory");  // the 256 epilogue threads
    }
    const bool have_acc = mbar_wait(&acc_full, (uint32_t)(tj & 1), &abort_flag, a.status, kLimit);
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    if (a.epi == EPI_FOLD) {
      // 1. the whole 128 x BN accumulator tile -> shared memory as int32 (rings are idle);
      //    row stride BN + 1 keeps the 32 rows of a warp in distinct banks
      constexpr int TS = BN + 1;
      int32_t* T = reinterpret_cast<int32_t*>(base);
      const int qf = warp & 3, cbegf = ((warp - 2) >> 2) * (BN / 2);
      for (int c0 = cbegf; c0 < cbegf + BN / 2; c0 += 32) {
        __syncwarp();
        uint32_t v[32];
        const uint32_t taddr = tmem + ((uint32_t)(32 * qf) << 16) + (uint32_t)c0;
        asm volatile(
            "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,"
            "%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
            : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
              "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15]),
              "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]),
              "=r"(v[24]), "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
            : "r"(taddr));
        asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
        int32_t* trow = T + (32 * qf + lane) * TS + c0;
#pragma unroll
        for (int j = 0; j < 32; ++j) trow[j] = acc_int<kA512>(v[j]);
      }
      const int rpg = (int)a.rpg, imgs = f_imgs, khw = f_khw, HW = f_HW;
      const int c_first = f_c0, nc = f_nc;
      const int32_t* tap_off = f_tap;
      const int32_t* csf = f_csf;
      const float* s_scale = f_scale;
      const float* s_zero = f_zero;
      const int32_t* s_n = f_n;
      const int tt = threadIdx.x - 64;
      asm volatile("bar.sync 1, 256;" ::: "memory");  // the 256 epilogue threads
      // Folder: dx[n, c, h, w] = S'_n sum(acc taps) + Z'_n sum(colsum taps); entries of fcb
      // channels per sample (a last, narrower channel block skips the missing ones)
      const bool fixed_pos = fold_same3(a) && 256 % HW == 0;
      if (fixed_pos && have_acc) {
        // 3 x 3, stride 1, pad 1 with H W dividing 256: one input position per thread, its tap
        // offsets (tile row pos + (1 - i) W + (1 - j), column 3 i + j) and validity computed
        // once; the 9 shared loads of an output are independent (a tap outside reads offset 0
        // and is masked)
        const int pos = tt & (HW - 1);
        const int h = (int)a.fd_w.div((uint32_t)pos), w = pos - h * a.fW;
        int off[9];
        uint32_t msk = 0;
#pragma unroll
        for (int t = 0; t < 9; ++t) {
          const int di = 1 - t / 3, dj = 1 - t % 3;
          const bool v = (unsigned)(h + di) < (unsigned)a.fH && (unsigned)(w + dj) < (unsigned)a.fW;
          off[t] = v ? (di * a.fW + dj) * TS + t : 0;
          msk |= v ? 1u << t : 0u;
        }
        // two channels per iteration: their 18 shared loads are issued before either sum
        const int cstep = 256 / HW;
        for (int img = 0; img < imgs; ++img) {
          const int n = s_n[img];
          if (n < 0) break;
          const float sc = s_scale[img], ze = s_zero[img];
          for (int cl = tt / HW; cl < nc; cl += 2 * cstep) {
            const int cl2 = cl + cstep < nc ? cl + cstep : cl;  // a lone last channel is summed twice
            const int32_t* tp = T + (img * rpg + pos) * TS + cl * 9;
            const int32_t* tp2 = T + (img * rpg + pos) * TS + cl2 * 9;
            int32_t v[9], v2[9];
#pragma unroll
            for (int t = 0; t < 9; ++t) { v[t] = tp[off[t]]; v2[t] = tp2[off[t]]; }
            const int32_t cf = csf[cl * HW + pos], cf2 = csf[cl2 * HW + pos];
            int32_t acc = 0, acc2 = 0;
#pragma unroll
            for (int t = 0; t < 9; ++t) {
              acc += (msk >> t) & 1u ? v[t] : 0;
              acc2 += (msk >> t) & 1u ? v2[t] : 0;
            }
            // channel cl of this input position: NCHW stride H W, NHWC stride 1
            float* yo = kNhwc ? a.y + ((int64_t)n * HW + pos) * a.fC + c_first
                                : a.y + ((int64_t)n * a.fC + c_first) * HW + pos;
            const int64_t cst = kNhwc ? 1 : HW;
            yo[cl * cst] = __fadd_rn(__fmul_rn(sc, (float)acc), __fmul_rn(ze, (float)cf));
            if (cl2 != cl) yo[cl2 * cst] = __fadd_rn(__fmul_rn(sc, (float)acc2), __fmul_rn(ze, (float)cf2));
          }
        }
      }
      const int per_img = a.fcb * HW;
      for (int e = tt; !fixed_pos && have_acc && e < imgs * per_img; e += 256) {
        const int img = (int)a.fd_cbhw.div((uint32_t)e), rem = e - img * per_img;
        const int n = s_n[img];
        if (n < 0) break;
        const int cl = (int)a.fd_hw.div((uint32_t)rem), pos = rem - cl * HW;
        if (cl >= nc) continue;
        const int32_t* tim = T + img * rpg * TS + cl * khw;
        const int32_t* to = tap_off + pos * khw;
        int32_t acc = 0;
        if (fold_same3(a)) {
          // 3 x 3, stride 1, pad 1: tap (i, j) of input (h, w) is the product of output pixel
          // (h + 1 - i, w + 1 - j), i.e. tile row pos + (1 - i) W + (1 - j), column 3 i + j
          const int h = (int)a.fd_w.div((uint32_t)pos), w = pos - h * a.fW;
          const int32_t* tp = tim + pos * TS;
#pragma unroll
          for (int t = 0; t < 9; ++t) {
            const int di = 1 - t / 3, dj = 1 - t % 3;
            const bool v = (unsigned)(h + di) < (unsigned)a.fH && (unsigned)(w + dj) < (unsigned)a.fW;
            acc += v ? tp[(di * a.fW + dj) * TS + t] : 0;
          }
        } else if (khw == 9) {  // other 3 x 3 kernels: all table and tile loads in flight together
          int o[9];
#pragma unroll
          for (int t = 0; t < 9; ++t) o[t] = to[t];
#pragma unroll
          for (int t = 0; t < 9; ++t) acc += o[t] >= 0 ? tim[o[t]] : 0;
        } else {
          for (int t = 0; t < khw; ++t) {
            const int o = to[t];
            if (o >= 0) acc += tim[o];
          }
        }
        const float v = __fadd_rn(__fmul_rn(s_scale[img], (float)acc), __fmul_rn(s_zero[img], (float)csf[rem]));
        if (kNhwc)
          a.y[((int64_t)n * HW + pos) * a.fC + c_first + cl] = v;
        else
          a.y[((int64_t)n * a.fC + c_first + cl) * HW + pos] = v;
      }
      // the bulk stores of zeros must have read the zero buffer before the CTA exits
      if (fold_zero_issued) asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
    } else {
    const int q = warp & 3;                         // TMEM lane quarter of this warp
    // its share of the accumulator columns: the tile's 32-column chunks below N (all BN for the
    // cluster reduction, which reads every column of its partial tiles), the first half to warps
    // 2..5 and the rest to warps 6..9, so that a tile narrower than BN (64 output channels)
    // still spreads its epilogue over all eight warps (at most BN / 64 chunks per warp)
    const int nchunks = a.epi == EPI_CRED ? BN / 32 : (int)min((int64_t)(BN / 32), (a.N - n0 + 31) / 32);
    const int half = (nchunks + 1) >> 1;
    const int cbeg = (warp >= 6 ? half : 0) * 32, cend = (warp >= 6 ? nchunks : half) * 32;
    uint32_t* stage = reinterpret_cast<uint32_t*>(base) + (warp - 2) * 1024;  // 4 KB per warp (operand ring is idle)
    const int64_t row_base = m0 + 32 * q;
    for (int c0 = cbeg; c0 < cend; c0 += 32) {
      // accumulator columns past N hold no output (warp-uniform; the cluster reduction reads
      // every column of its partial tiles)
      if (a.epi != EPI_CRED && n0 + c0 >= a.N) break;
      __syncwarp();
      uint32_t v[32];
      const uint32_t taddr = tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)c0;
      asm volatile(
          "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,"
          "%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
          : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
            "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15]),
            "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]),
            "=r"(v[24]), "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
          : "r"(taddr));
      asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
      if (a.epi == EPI_CRED) {
        // this CTA's partial sums -> its shared tile, read by the whole cluster below
        const int r = 32 * q + lane;
#pragma unroll
        for (int c = 0; c < 8; ++c) {
          int4 w;
          w.x = acc_int<kA512>(v[4 * c + 0]);
          w.y = acc_int<kA512>(v[4 * c + 1]);
          w.z = acc_int<kA512>(v[4 * c + 2]);
          w.w = acc_int<kA512>(v[4 * c + 3]);
          *reinterpret_cast<int4*>(base + ptile_off(r, (c0 >> 2) + c)) = w;
        }
        continue;
      }
      if (!have_acc) continue;
      if (a.tma_out && row_base + 32 <= valid_rows) {
        // stage the warp's 32 x 32 block (row = lane; 16-byte chunk c of a row at chunk
        // c ^ (row & 7), the 128-byte swizzle of the output maps), then one TMA store per
        // output; TMA clips columns past the tensor
        // 8 KB per warp and 32-column chunk (y then acc): no wait between the warp's chunks
        // (SHORT tiles store y alone: 4 KB per chunk, within the smaller ring)
        unsigned char* stg = SHORT ? base + (warp - 2) * 8192 + ((c0 - cbeg) >> 5) * 4096
                                   : base + (warp - 2) * 16384 + ((c0 - cbeg) >> 5) * 8192;
        float* sy = reinterpret_cast<float*>(stg);
        int32_t* sacc = reinterpret_cast<int32_t*>(stg + 4096);
        const int64_t nb = n0 + c0;
#pragma unroll
        for (int c = 0; c < 8; ++c) {
          const int32_t i0 = acc_int<kA512>(v[4 * c + 0]);
          const int32_t i1 = acc_int<kA512>(v[4 * c + 1]);
          const int32_t i2 = acc_int<kA512>(v[4 * c + 2]);
          const int32_t i3 = acc_int<kA512>(v[4 * c + 3]);
          const int off = lane * 32 + ((c ^ (lane & 7)) << 2);
          if (a.tma_out & 1) {
            const float4 g4 = *reinterpret_cast<const float4*>(gamma_s + c0 + 4 * c);
            float4 y4 = make_float4(__fmul_rn(g4.x, (float)i0), __fmul_rn(g4.y, (float)i1),
                                    __fmul_rn(g4.z, (float)i2), __fmul_rn(g4.w, (float)i3));
            if (a.bias) {
              const float4 b4 = *reinterpret_cast<const float4*>(bias_s + c0 + 4 * c);
              y4 = make_float4(__fadd_rn(y4.x, b4.x), __fadd_rn(y4.y, b4.y), __fadd_rn(y4.z, b4.z),
                               __fadd_rn(y4.w, b4.w));
            }
            *reinterpret_cast<float4*>(sy + off) = y4;
          }
          if (a.tma_out & 2) *reinterpret_cast<int4*>(sacc + off) = make_int4(i0, i1, i2, i3);
        }
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        __syncwarp();
        if (lane == 0) {
          if (a.tma_out & 1) tma_store_2d(&tmY, sy, (int)nb, (int)row_base);
          if (a.tma_out & 2) tma_store_2d(&tmAcc, sacc, (int)nb, (int)row_base);
          asm volatile("cp.async.bulk.commit_group;" ::: "memory");
        }
        continue;
      }
      if (a.epi == EPI_ACC32 && a.acc_cm) {
        // column-major: lane = row, so each column's 32 rows leave as one coalesced line
        const int64_t r = row_base + lane;
        const bool rv = r < valid_rows && r < a.M;
        int32_t* dst = a.acc + (n0 + c0) * a.ldo + r;
        const int64_t ncol = a.N - (n0 + c0);  // > 0 here
        if (a.acc_cm == 2) {
          int16_t* dst16 = reinterpret_cast<int16_t*>(a.acc) + (n0 + c0) * a.ldo + r;
#pragma unroll
          for (int j = 0; j < 32; ++j)
            if (rv && j < ncol) dst16[j * a.ldo] = (int16_t)acc_int<kA512>(v[j]);
          continue;
        }
#pragma unroll
        for (int j = 0; j < 32; ++j)
          if (rv && j < ncol) dst[j * a.ldo] = acc_int<kA512>(v[j]);
        continue;
      }
      if (a.epi == EPI_ACC32) {
        // the int32 accumulators through the warp's 4 KB staging block (row = lane, word j at
        // j ^ lane), then one coalesced 128-byte row segment per store (lanes over columns)
        // instead of each lane writing its own row
        __syncwarp();  // the previous chunk's reads of the block are done
#pragma unroll
        for (int j = 0; j < 32; ++j) stage[lane * 32 + (j ^ lane)] = (uint32_t)acc_int<kA512>(v[j]);
        __syncwarp();
        const int64_t col = n0 + c0 + lane;
        const int64_t left = (valid_rows < a.M ? valid_rows : a.M) - row_base;
        const int rows = left <= 0 ? 0 : (left >= 32 ? 32 : (int)left);
        if (col < a.N) {
          int32_t* dst = a.acc + row_base * a.ldo + col;
          for (int rr = 0; rr < rows; ++rr) dst[rr * a.ldo] = (int32_t)stage[rr * 32 + (lane ^ rr)];
        }
        continue;
      }
      if (a.epi != EPI_RED) {
        // direct stores: this thread's row, 32 consecutive columns
        const int64_t r = row_base + lane;
        const int64_t nb = n0 + c0;
        if (r >= valid_rows || r >= a.M || nb >= a.N) continue;
        int32_t iv[32];
#pragma unroll
        for (int j = 0; j < 32; ++j) iv[j] = acc_int<kA512>(v[j]);
        const bool full = nb + 32 <= a.N && (a.ldo % 4) == 0;
        int64_t out_row = r;
        float sc = 0.f, ze = 0.f;
        if (a.epi == EPI_DX) {
          const int64_t slot = r / a.rpg;
          out_row = (int64_t)__ldg(a.kept_idx + slot) * a.rpg + (r - slot * a.rpg);
          sc = __ldg(a.scale + slot);
          ze = __ldg(a.zero + slot);
        }
        if (a.epi == EPI_FWD && !a.y) {  // the integer accumulators alone
          int32_t* orow = a.acc + out_row * a.ldo + nb;
          if (full) {
#pragma unroll
            for (int j = 0; j < 32; j += 4) *reinterpret_cast<int4*>(orow + j) = make_int4(iv[j], iv[j + 1], iv[j + 2], iv[j + 3]);
          } else {
            for (int j = 0; j < 32 && nb + j < a.N; ++j) orow[j] = iv[j];
          }
        } else if (a.epi == EPI_FWD) {
          float* yrow = a.y + out_row * a.ldo + nb;
          if (full) {
#pragma unroll
            for (int j = 0; j < 32; j += 4) {
              const float4 g4 = __ldg(reinterpret_cast<const float4*>(a.gamma + nb + j));
              float4 y4 = make_float4(__fmul_rn(g4.x, (float)iv[j]), __fmul_rn(g4.y, (float)iv[j + 1]),
                                      __fmul_rn(g4.z, (float)iv[j + 2]), __fmul_rn(g4.w, (float)iv[j + 3]));
              if (a.bias) {
                const float4 b4 = __ldg(reinterpret_cast<const float4*>(a.bias + nb + j));
                y4 = make_float4(__fadd_rn(y4.x, b4.x), __fadd_rn(y4.y, b4.y), __fadd_rn(y4.z, b4.z),
                                 __fadd_rn(y4.w, b4.w));
              }
              *reinterpret_cast<float4*>(yrow + j) = y4;
              if (a.acc)
                *reinterpret_cast<int4*>(a.acc + out_row * a.ldo + nb + j) = make_int4(iv[j], iv[j + 1], iv[j + 2], iv[j + 3]);
            }
          } else {
            for (int j = 0; j < 32 && nb + j < a.N; ++j) {
              const float g = __fmul_rn(__ldg(a.gamma + nb + j), (float)iv[j]);
              yrow[j] = a.bias ? __fadd_rn(g, __ldg(a.bias + nb + j)) : g;
              if (a.acc) a.acc[out_row * a.ldo + nb + j] = iv[j];
            }
          }
        } else if (a.epi == EPI_ACC32) {
          int32_t* orow = a.acc + out_row * a.ldo + nb;
          if (full) {
#pragma unroll
            for (int j = 0; j < 32; j += 4) *reinterpret_cast<int4*>(orow + j) = make_int4(iv[j], iv[j + 1], iv[j + 2], iv[j + 3]);
          } else {
            for (int j = 0; j < 32 && nb + j < a.N; ++j) orow[j] = iv[j];
          }
        } else {  // EPI_DX
          float* orow = a.y + out_row * a.ldo + nb;
          if (full) {
#pragma unroll
            for (int j = 0; j < 32; j += 4) {
              const int4 c4 = __ldg(reinterpret_cast<const int4*>(a.cs + nb + j));
              *reinterpret_cast<float4*>(orow + j) = make_float4(
                  __fadd_rn(__fmul_rn(sc, (float)iv[j + 0]), __fmul_rn(ze, (float)c4.x)),
                  __fadd_rn(__fmul_rn(sc, (float)iv[j + 1]), __fmul_rn(ze, (float)c4.y)),
                  __fadd_rn(__fmul_rn(sc, (float)iv[j + 2]), __fmul_rn(ze, (float)c4.z)),
                  __fadd_rn(__fmul_rn(sc, (float)iv[j + 3]), __fmul_rn(ze, (float)c4.w)));
            }
          } else {
            for (int j = 0; j < 32 && nb + j < a.N; ++j)
              orow[j] = __fadd_rn(__fmul_rn(sc, (float)iv[j]), __fmul_rn(ze, (float)__ldg(a.cs + nb + j)));
          }
        }
        continue;
      }
      // split-K reduction: stage the 32 x 32 block (row `lane`, 16-byte chunk c stored at
      // chunk c ^ (lane & 7)), then add one coalesced 128-byte row per instruction
#pragma unroll
      for (int c = 0; c < 8; ++c) {
        uint4 w;
        w.x = (uint32_t)acc_int<kA512>(v[4 * c + 0]);
        w.y = (uint32_t)acc_int<kA512>(v[4 * c + 1]);
        w.z = (uint32_t)acc_int<kA512>(v[4 * c + 2]);
        w.w = (uint32_t)acc_int<kA512>(v[4 * c + 3]);
        *reinterpret_cast<uint4*>(stage + lane * 32 + ((c ^ (lane & 7)) << 2)) = w;
      }
      __syncwarp();
      const int64_t n = n0 + c0 + lane;  // this lane's column
      if (n < a.N) {
#pragma unroll 4
        for (int rr = 0; rr < 32; ++rr) {
          const int64_t r = row_base + rr;
          if (r >= valid_rows || r >= a.M) break;
          atomicAdd(a.acc + r * a.ldo + n, (int32_t)stage[rr * 32 + ((((lane >> 2) ^ (rr & 7))) << 2) + (lane & 3)]);
        }
      }
    }
    // the stores must have read the staging buffers before the CTA exits
    if (a.tma_out && lane == 0) asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
    }  // epilogue modes other than EPI_FOLD
    if (kPersist) {
      // every epilogue warp has read its staging block and its accumulator columns before the
      // next tile's operands go into the ring (also by TMA) and its products into TMEM
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      __syncwarp();
      asm volatile("bar.sync 1, 256;" ::: "memory");
    }
  }
  gbase += nk;
  }  // output tiles
  if (warp == 0 && lane == 0) {
    // drain: every issued copy must land before the CTA may exit
    for (int i = (issued > RS ? issued - RS : 0); i < issued; ++i) {
      const int s = i % RS, it = i / RS;
      const uint64_t t0 = gtimer();
      while (!mbar_test(&raw_full[s], it & 1) && gtimer() - t0 < kWaitNs) {
      }
    }
  }

  // The producer and MMA roles ran on lane 0 only; reconverge before the aligned barriers
  // (the cluster's, and the one that orders the epilogue's TMEM reads before warp 1 frees TMEM).
  __syncwarp();
  if (a.epi == EPI_CRED) {
    // every CTA of the cluster reaches both barriers, also after an expired wait
    const uint32_t rank = cluster_rank(), nr = cluster_size();
    const bool vec = (a.ldo % 4) == 0;
    if (blockIdx.y == 0) {
      // pruned channels (independent of the products, so before the cluster barrier): zero
      // rows of dw over this tile's columns, shared by the cluster; the slots of a thread's
      // next 4 elements are loaded together first
      const int64_t step = (int64_t)nr * kThreads;
      for (int64_t e0 = (int64_t)rank * kThreads + threadIdx.x; e0 < a.D * 32; e0 += 4 * step) {
        int32_t sl[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) sl[u] = __ldg(a.slot_of_group + (min(e0 + u * step, a.D * 32 - 1) >> 5));
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int64_t e = e0 + u * step;
          const int64_t j = e >> 5, n = n0 + 4 * (e & 31);
          if (e >= a.D * 32 || n >= a.N || sl[u] >= 0) continue;
          float* wrow = a.y + j * a.ldo + n;
          if (vec && n + 4 <= a.N) *reinterpret_cast<float4*>(wrow) = make_float4(0.f, 0.f, 0.f, 0.f);
          else for (int t = 0; t < 4 && n + t < a.N; ++t) wrow[t] = 0.f;
        }
      }
    }
    // the tile rows that exist (up to the capacity) are divided over the cluster's CTAs
    const int64_t rows_here = a.M - m0;
    const int nrows = rows_here >= kBM ? kBM : (rows_here <= 0 ? 0 : (int)rows_here);
    const int rpr = (nrows + (int)nr - 1) / (int)nr;  // tile rows summed by each CTA
    const int r_lo = min(nrows, (int)rank * rpr), r_hi = min(nrows, r_lo + rpr);
    const int nel = (r_hi - r_lo) * 32;
    // the row and column inputs of the dequantization (kept channel, S', Z', column sums of
    // sign(X)) of a chunk, loaded together from clamped indices; the first chunk's before
    // the cluster barrier
    int64_t kj = 0;
    float ksc = 0.f, kze = 0.f;
    int32_t kcs[4] = {0, 0, 0, 0};
    auto chunk_inputs = [&](int e) {
      const int64_t grow = min(m0 + r_lo + (e >> 5), a.M - 1), n = n0 + 4 * (e & 31);
      kj = __ldg(a.kept_idx + grow);
      ksc = __ldg(a.scale + grow);
      kze = __ldg(a.zero + grow);
#pragma unroll
      for (int t = 0; t < 4; ++t) kcs[t] = __ldg(a.cs + min(n + t, a.N - 1));
    };
    if ((int)threadIdx.x < nel) chunk_inputs(threadIdx.x);
    cluster_sync_all();
    const uint32_t pbase = smem_u32(base);
    const bool ok = !abort_flag;
    for (int e = threadIdx.x; e < nel; e += kThreads) {
      if (e != (int)threadIdx.x) chunk_inputs(e);
      const int r = r_lo + (e >> 5), ch = e & 31;
      const int64_t grow = m0 + r, n = n0 + 4 * ch;
      if (grow >= a.M || n >= a.N) continue;
      int4 sum = make_int4(0, 0, 0, 0);
      const bool kept = ok && grow < valid_rows;
      if (kept) {
        // all of the cluster's partial chunks in flight together (clusters have <= 8 CTAs)
        int4 t[8];
#pragma unroll
        for (uint32_t src = 0; src < 8; ++src)
          if (src < nr) t[src] = ld_cluster_v4(pbase + ptile_off(r, ch), src);
#pragma unroll
        for (uint32_t src = 0; src < 8; ++src)
          if (src < nr) { sum.x += t[src].x; sum.y += t[src].y; sum.z += t[src].z; sum.w += t[src].w; }
      }
      const int32_t sv[4] = {sum.x, sum.y, sum.z, sum.w};
      int32_t* arow = a.acc + grow * a.ldo + n;
      if (vec && n + 4 <= a.N) *reinterpret_cast<int4*>(arow) = sum;
      else for (int t = 0; t < 4 && n + t < a.N; ++t) arow[t] = sv[t];
      if (kept) {
        float* wrow = a.y + kj * a.ldo + n;
        float o[4];
#pragma unroll
        for (int t = 0; t < 4; ++t)
          o[t] = n + t < a.N ? __fadd_rn(__fmul_rn(ksc, (float)sv[t]), __fmul_rn(kze, (float)kcs[t])) : 0.f;
        if (vec && n + 4 <= a.N) *reinterpret_cast<float4*>(wrow) = make_float4(o[0], o[1], o[2], o[3]);
        else for (int t = 0; t < 4 && n + t < a.N; ++t) wrow[t] = o[t];
      }
    }
    cluster_sync_all();  // no CTA leaves while another still reads its tile
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (warp == 1) {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(S::kTmemCols));
  }
}

// ------------------------------------------------------------------ host side
// The driver's tensor-map encoder, looked up once (a function-local static: its initialisation
// is thread-safe, so host threads that launch concurrently never race on it).
static PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static const PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    return static_cast<PFN_cuTensorMapEncodeTiled_v12000>(nullptr);
  }();
  return fn;
}

// 2-D map of a row-major matrix: inner extent `cols` elements, `rows` rows, row stride `ld_bytes`.
static bool make_map(CUtensorMap* m, const void* ptr, CUtensorMapDataType type, int64_t cols, int64_t rows,
                     int64_t ld_bytes, uint32_t box_cols, uint32_t box_rows, CUtensorMapSwizzle swz_mode) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)ld_bytes};
  cuuint32_t box[2] = {box_cols, box_rows};
  cuuint32_t estr[2] = {1, 1};
  return fn(m, type, 2, const_cast<void*>(ptr), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swz_mode,
            CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// SMs of the current device (cached per device ordinal).
static int sm_count() {
  static std::atomic<int> cache[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 152;
  int n = cache[dev].load(std::memory_order_relaxed);
  if (n > 0) return n;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1) n = 152;
  cache[dev].store(n, std::memory_order_relaxed);
  return n;
}

// Output tiles of a launch and the resident CTAs of one wave (1 per SM, 2 for SHORT tiles).
static int64_t out_tiles(const TcArgs& a, int bn) { return ((a.N + bn - 1) / bn) * ((a.M + kBM - 1) / kBM); }
static int64_t tile_wave(bool short_tile) { return (int64_t)sm_count() * (short_tile ? 2 : 1); }

template <bool A_CODES, bool BITS8, int BN, bool SHORT = false, int X = 0>
static cudaError_t launch_tc(const CUtensorMap& ma, const CUtensorMap& mb, const TcArgs& a_in, int splits,
                             cudaStream_t s, const CUtensorMap* my = nullptr, const CUtensorMap* macc = nullptr,
                             bool cluster = false) {
  static const CUtensorMap unused{};  // never read: the matching tma_out bit is clear
  using S = TcSmem<A_CODES, BITS8, BN, SHORT, (X & 64) == 0>;
  static std::atomic<uint64_t> attr{0};
  const cudaError_t ea = smem_attr_once((const void*)tc_gemm_kernel<A_CODES, BITS8, BN, SHORT, X>, S::kBytes, attr);
  if (ea != cudaSuccess) return ea;
  TcArgs a = a_in;
  dim3 grid((unsigned)(a.grid_x > 0 ? a.grid_x : (a.N + BN - 1) / BN), (unsigned)((a.M + kBM - 1) / kBM),
            (unsigned)splits);
  if constexpr ((X & 128) != 0) {  // persistent: one wave of CTAs over all output tiles
    a.p_tiles_n = (a.N + BN - 1) / BN;
    a.p_tiles = out_tiles(a, BN);
    grid = dim3((unsigned)std::min<int64_t>(a.p_tiles, tile_wave(SHORT)), 1, 1);
  }
  if (cluster)
    launch_k_cluster(tc_gemm_kernel<A_CODES, BITS8, BN, SHORT, X>, dim3(grid), dim3(kThreads), S::kBytes, s,
                     (unsigned)splits, ma, mb, my ? *my : unused, macc ? *macc : unused, a);
  else
    launch_k(tc_gemm_kernel<A_CODES, BITS8, BN, SHORT, X>, dim3(grid), dim3(kThreads), S::kBytes, s, ma, mb,
             my ? *my : unused, macc ? *macc : unused, a);
  fqt1_count_launches(1);
  return cudaGetLastError();
}

// Forward with a prepared A map: B = sign(W) rows [D][words(K)]; a carries the implicit-
// convolution fields (impl = 0 for a plain A = sign(X) rows map).
static cudaError_t launch_fwd_common(const CUtensorMap& ma, TcArgs a, const uint32_t* B, int64_t M, int64_t D,
                                     int64_t K, const float* gamma, const float* bias, int32_t* acc, float* y,
                                     int32_t* status, cudaStream_t s, const uint8_t* Be = nullptr, int64_t ldbe = 0,
                                     bool implicit = false) {
  using S = TcSmem<false, false, 128>;
  const int64_t ldw = fqt1_packed_words(K);
  CUtensorMap mb;
  if (Be) {  // e4m3 sign(W) rows [D][ldbe] bytes: 128 x 128 boxes, 128-byte swizzle
    if (!make_map(&mb, Be, CU_TENSOR_MAP_DATA_TYPE_UINT8, K, D, ldbe, kBK, 128, CU_TENSOR_MAP_SWIZZLE_128B))
      return cudaErrorInvalidValue;
  } else if (!make_map(&mb, B, CU_TENSOR_MAP_DATA_TYPE_UINT32, ldw, D, ldw * 4, 4 * S::KSUB, 128,
                       CU_TENSOR_MAP_SWIZZLE_NONE)) {
    return cudaErrorInvalidValue;
  }
  a.M = M; a.N = D; a.L = K; a.count = nullptr; a.rows_per_count = 1;
  a.k_tiles = (int)((K + kBK * S::KSUB - 1) / (kBK * S::KSUB)); a.tiles_per_split = a.k_tiles;
  a.epi = EPI_FWD; a.gamma = gamma; a.bias = bias; a.y = y; a.acc = acc; a.ldo = D; a.status = status;
  // outputs leave through TMA stores when their rows are 16-byte multiples (y may be null: the
  // integer accumulators alone)
  CUtensorMap my{}, macc{};
  if (D % 4 == 0) {
    bool ok = true;
    if (y) ok = make_map(&my, y, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, D, M, D * 4, 32, 32, CU_TENSOR_MAP_SWIZZLE_128B);
    if (ok && acc)
      ok = make_map(&macc, acc, CU_TENSOR_MAP_DATA_TYPE_INT32, D, M, D * 4, 32, 32, CU_TENSOR_MAP_SWIZZLE_128B);
    if (ok) a.tma_out = (y ? 1 : 0) | (acc ? 2 : 0);
  }
  if (implicit) return launch_tc<false, false, 128, false, 1>(ma, mb, a, 1, s, &my, &macc);
  // one operand stage without int32 outputs (tall, short layers such as the 7 x 7 stem): SHORT
  // tiles, two CTAs per SM, so that one CTA's set-up and epilogue overlap the other's products
  // more output tiles than one wave of CTAs: persistent CTAs over the tiles (mode bit 7)
  const bool short_tile = a.k_tiles == 1 && !acc;
  const bool persist = out_tiles(a, 128) > tile_wave(short_tile);
  if (Be) {
    if (short_tile && persist) return launch_tc<false, false, 128, true, 2 | 64 | 128>(ma, mb, a, 1, s, &my, &macc);
    if (short_tile) return launch_tc<false, false, 128, true, 2 | 64>(ma, mb, a, 1, s, &my, &macc);
    if (persist) return launch_tc<false, false, 128, false, 2 | 128>(ma, mb, a, 1, s, &my, &macc);
    return launch_tc<false, false, 128, false, 2>(ma, mb, a, 1, s, &my, &macc);
  }
  if (short_tile && persist) return launch_tc<false, false, 128, true, 64 | 128>(ma, mb, a, 1, s, &my, &macc);
  if (short_tile) return launch_tc<false, false, 128, true, 64>(ma, mb, a, 1, s, &my, &macc);
  if (persist) return launch_tc<false, false, 128, false, 128>(ma, mb, a, 1, s, &my, &macc);
  return launch_tc<false, false, 128>(ma, mb, a, 1, s, &my, &macc);
}

// Forward: A = sign(X) rows [M][words(K)], B = sign(W) rows [D][words(K)].
cudaError_t launch_fwd_tc(const uint32_t* A, const uint32_t* B, int64_t M, int64_t D, int64_t K, const float* gamma,
                          const float* bias, int32_t* acc, float* y, int32_t* status, cudaStream_t s) {
  using S = TcSmem<false, false, 128>;
  const int64_t ldw = fqt1_packed_words(K);
  CUtensorMap ma;
  if (!make_map(&ma, A, CU_TENSOR_MAP_DATA_TYPE_UINT32, ldw, M, ldw * 4, 4 * S::KSUB, kBM,
                CU_TENSOR_MAP_SWIZZLE_NONE))
    return cudaErrorInvalidValue;
  return launch_fwd_common(ma, TcArgs{}, B, M, D, K, gamma, bias, acc, y, status, s);
}

// The failure-path test: fqt1_fwd_gemm's kernel with one operand-stage arrive withheld (bit 4).
cudaError_t launch_fwd_lost_arrive_tc(const uint32_t* A, const uint32_t* B, int64_t M, int64_t D, int64_t K,
                                      const float* gamma, float* y, int32_t* status, cudaStream_t s) {
  using S = TcSmem<false, false, 128>;
  const int64_t ldw = fqt1_packed_words(K);
  CUtensorMap ma, mb;
  if (!make_map(&ma, A, CU_TENSOR_MAP_DATA_TYPE_UINT32, ldw, M, ldw * 4, 4 * S::KSUB, kBM,
                CU_TENSOR_MAP_SWIZZLE_NONE) ||
      !make_map(&mb, B, CU_TENSOR_MAP_DATA_TYPE_UINT32, ldw, D, ldw * 4, 4 * S::KSUB, 128,
                CU_TENSOR_MAP_SWIZZLE_NONE))
    return cudaErrorInvalidValue;
  TcArgs a{};
  a.M = M; a.N = D; a.L = K; a.count = nullptr; a.rows_per_count = 1;
  a.k_tiles = (int)((K + kBK * S::KSUB - 1) / (kBK * S::KSUB)); a.tiles_per_split = a.k_tiles;
  a.epi = EPI_FWD; a.gamma = gamma; a.y = y; a.ldo = D; a.status = status;
  return launch_tc<false, false, 128, false, 16>(ma, mb, a, 1, s);
}

// Forward with B = e4m3 sign(W) rows [D][ldbe] bytes (ldbe a multiple of 16, bytes past K zero).
cudaError_t launch_fwd_e4m3w_tc(const uint32_t* A, const uint8_t* Be, int64_t ldbe, int64_t M, int64_t D, int64_t K,
                                const float* gamma, const float* bias, int32_t* acc, float* y, int32_t* status,
                                cudaStream_t s) {
  using S = TcSmem<false, false, 128>;
  const int64_t ldw = fqt1_packed_words(K);
  CUtensorMap ma;
  if (!make_map(&ma, A, CU_TENSOR_MAP_DATA_TYPE_UINT32, ldw, M, ldw * 4, 4 * S::KSUB, kBM,
                CU_TENSOR_MAP_SWIZZLE_NONE))
    return cudaErrorInvalidValue;
  return launch_fwd_common(ma, TcArgs{}, nullptr, M, D, K, gamma, bias, acc, y, status, s, Be, ldbe);
}

// Forward with A = e4m3 sign(X_u) rows [M][ldxe] and B = e4m3 sign(W) rows [D][ldbe] (bytes
// +1 = 0x38, -1 = 0xB8): both operands go by TMA straight into the MMA, nothing is expanded.
cudaError_t launch_fwd_e4m3x_tc(const uint8_t* Xe, int64_t ldxe, const uint8_t* Be, int64_t ldbe, int64_t M, int64_t D,
                                int64_t K, const float* gamma, const float* bias, int32_t* acc, float* y,
                                int32_t* status, cudaStream_t s) {
  CUtensorMap ma, mb;
  if (!make_map(&ma, Xe, CU_TENSOR_MAP_DATA_TYPE_UINT8, K, M, ldxe, kBK, kBM, CU_TENSOR_MAP_SWIZZLE_128B) ||
      !make_map(&mb, Be, CU_TENSOR_MAP_DATA_TYPE_UINT8, K, D, ldbe, kBK, 128, CU_TENSOR_MAP_SWIZZLE_128B))
    return cudaErrorInvalidValue;
  TcArgs a{};
  a.M = M; a.N = D; a.L = K; a.count = nullptr; a.rows_per_count = 1;
  a.k_tiles = (int)((K + kCodesStageK - 1) / kCodesStageK); a.tiles_per_split = a.k_tiles;
  a.epi = EPI_FWD; a.gamma = gamma; a.bias = bias; a.y = y; a.acc = acc; a.ldo = D; a.status = status;
  CUtensorMap my{}, macc{};
  if (D % 4 == 0) {
    bool ok = true;
    if (y) ok = make_map(&my, y, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, D, M, D * 4, 32, 32, CU_TENSOR_MAP_SWIZZLE_128B);
    if (ok && acc)
      ok = make_map(&macc, acc, CU_TENSOR_MAP_DATA_TYPE_INT32, D, M, D * 4, 32, 32, CU_TENSOR_MAP_SWIZZLE_128B);
    if (ok) a.tma_out = (y ? 1 : 0) | (acc ? 2 : 0);
  }
  if (a.k_tiles <= 2 && !acc) return launch_tc<true, false, 128, true, 2 | 32 | 64>(ma, mb, a, 1, s, &my, &macc);
  return launch_tc<true, false, 128, false, 2 | 32>(ma, mb, a, 1, s, &my, &macc);
}

// Implicit-GEMM forward of a stride-1 "same" convolution (kh = kw = 2 pad + 1, C a multiple of
// 128).  A tile of 128 output pixels is whole images (H W divides 128) or whole image rows (W
// divides 128 and the rows of a tile divide H); its A sub-tiles are 4-D boxes of the pixel-major
// sign words xp [N][H][W][C / 32], one per (tap, 128 channels).  B = tap-major sign(W) rows.
bool implicit_conv_supported(int64_t N, int64_t C, int64_t H, int64_t W, int64_t kh, int64_t kw, int64_t stride,
                             int64_t pad) {
  if (N < 1 || C < 1 || H < 1 || W < 1 || stride != 1 || kh != kw || kh != 2 * pad + 1 || C % 128 != 0) return false;
  if (C * kh * kw >= (1ll << 24) || N * H * W >= (1ll << 31) || (N * H * W + kBM - 1) / kBM > 65535) return false;
  const int64_t HW = H * W;
  if (HW <= kBM) return kBM % HW == 0;
  return W <= kBM && kBM % W == 0 && H % (kBM / W) == 0;
}

cudaError_t launch_fwd_implicit_tc(const uint32_t* xp, const uint32_t* wt, int N, int C, int H, int W, int k, int pad,
                                   int64_t D, const float* gamma, const float* bias, int32_t* acc, float* y,
                                   int32_t* status, cudaStream_t s) {
  auto fn = encode_fn();
  if (!fn) return cudaErrorInvalidValue;
  const int64_t cw = fqt1_packed_words(C), HW = (int64_t)H * W;
  const uint32_t box_h = HW <= kBM ? (uint32_t)H : (uint32_t)(kBM / W);
  const uint32_t box_n = HW <= kBM ? (uint32_t)(kBM / HW) : 1u;
  // sub-tiles per box: the largest power of two (<= KSUB) dividing the 128-channel blocks of a tap
  using S = TcSmem<false, false, 128>;
  int isb = 0;
  while ((1 << (isb + 1)) <= S::KSUB && (C / 128) % (1 << (isb + 1)) == 0) ++isb;
  cuuint64_t dims[4] = {(cuuint64_t)cw, (cuuint64_t)W, (cuuint64_t)H, (cuuint64_t)N};
  cuuint64_t strides[3] = {(cuuint64_t)(cw * 4), (cuuint64_t)(cw * 4 * W), (cuuint64_t)(cw * 4 * HW)};
  cuuint32_t box[4] = {4u << isb, (cuuint32_t)W, box_h, box_n};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  CUtensorMap ma;
  if (fn(&ma, CU_TENSOR_MAP_DATA_TYPE_UINT32, 4, const_cast<uint32_t*>(xp), dims, strides, box, estr,
         CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  TcArgs a{};
  a.iC = C; a.ikw = k; a.ikhw = k * k; a.ipad = pad; a.iW = W; a.iHW = (int)HW; a.isb = isb;
  return launch_fwd_common(ma, a, wt, (int64_t)N * HW, D, (int64_t)C * k * k, gamma, bias, acc, y, status, s,
                           nullptr, 0, true);
}

// Codes x signs: out[r, n] = sum_j Q[r, j] S[n, j], Q [rows][ld] uint8 (valid rows *count * rpc),
// S [n_s][words(L)] packed signs.  epi: EPI_ACC32 (store), EPI_RED (split-K add), EPI_DX (dequantize).
// Be (optional): S as e4m3 sign bytes [n_s][ldbe] instead of packed words, by TMA into the
// operand ring.
cudaError_t launch_codes_tc(int bits, const uint8_t* Q, int64_t ldq, int64_t max_rows, const int32_t* count,
                            int64_t rows_per_count, const uint32_t* Sg, int64_t n_s, int64_t L, int epi, int splits,
                            const TcArgs& epi_args, cudaStream_t s, const uint8_t* Be = nullptr, int64_t ldbe = 0) {
  const int64_t lds = fqt1_packed_words(L);
  CUtensorMap ma, mb;
  if (!make_map(&ma, Q, CU_TENSOR_MAP_DATA_TYPE_UINT8, L, max_rows, ldq, kBK, kBM, CU_TENSOR_MAP_SWIZZLE_128B))
    return cudaErrorInvalidValue;
  if (Be) {
    if (!make_map(&mb, Be, CU_TENSOR_MAP_DATA_TYPE_UINT8, L, n_s, ldbe, kBK, 128, CU_TENSOR_MAP_SWIZZLE_128B))
      return cudaErrorInvalidValue;
  } else if (!make_map(&mb, Sg, CU_TENSOR_MAP_DATA_TYPE_UINT32, lds, n_s, lds * 4, kCodesStageK / 32, 128,
                       CU_TENSOR_MAP_SWIZZLE_NONE)) {
    return cudaErrorInvalidValue;
  }
  TcArgs a = epi_args;
  a.M = max_rows; a.N = n_s; a.L = L; a.count = count; a.rows_per_count = rows_per_count;
  a.k_tiles = (int)((L + kCodesStageK - 1) / kCodesStageK);
  a.tiles_per_split = (a.k_tiles + splits - 1) / splits;
  a.epi = epi;
  const int z = (a.k_tiles + a.tiles_per_split - 1) / a.tiles_per_split;
  // short contractions per CTA (the grad_input product of layers with few output channels):
  // SHORT tiles, two CTAs per SM (their epilogues store directly, without TMA staging)
  const bool short_tile = a.tiles_per_split == 1 && !a.tma_out;
  if (Be) {
    if (bits == 8) return launch_tc<true, true, 128, false, 2>(ma, mb, a, z, s);
    const bool persist_b = short_tile && z == 1 && out_tiles(a, 128) > tile_wave(true);
    if (persist_b) return launch_tc<true, false, 128, true, 2 | 8 | 64 | 128>(ma, mb, a, z, s);
    if (short_tile) return launch_tc<true, false, 128, true, 2 | 8 | 64>(ma, mb, a, z, s);
    return launch_tc<true, false, 128, false, 2 | 8>(ma, mb, a, z, s);
  }
  if (bits == 8) return launch_tc<true, true, 128>(ma, mb, a, z, s);
  // more output tiles than one wave, without splits: persistent CTAs over the tiles (mode bit 7)
  const bool persist = z == 1 && out_tiles(a, 128) > tile_wave(short_tile);
  if (short_tile && persist) return launch_tc<true, false, 128, true, 8 | 64 | 128>(ma, mb, a, z, s);
  if (short_tile) return launch_tc<true, false, 128, true, 8 | 64>(ma, mb, a, z, s);
  if (persist) return launch_tc<true, false, 128, false, 8 | 128>(ma, mb, a, z, s);
  return launch_tc<true, false, 128, false, 8>(ma, mb, a, z, s);  // codes < 16: A straight from TMA
}

// grad_input of a convolution with the Folder in the epilogue (EPI_FOLD, 256-column tiles).
cudaError_t launch_fold_tc(int bits, const uint8_t* Q, int64_t ldq, int64_t max_rows, const int32_t* count,
                           const uint32_t* Sg, int64_t K, int64_t D, const int32_t* kept_idx, const float* scale,
                           const float* zero, const int32_t* cs, const int32_t* slot_of_group, float* dx, int N, int C,
                           int H, int W, int kh, int kw, int stride, int pad, int Ho, int Wo, int32_t* status,
                           cudaStream_t s, const uint8_t* Bte, int64_t ldbte, int nhwc) {
  const int64_t lds = fqt1_packed_words(D);
  CUtensorMap ma, mb;
  if (!make_map(&ma, Q, CU_TENSOR_MAP_DATA_TYPE_UINT8, D, max_rows, ldq, kBK, kBM, CU_TENSOR_MAP_SWIZZLE_128B))
    return cudaErrorInvalidValue;
  if (Bte) {  // e4m3 sign(W)^T rows [K][ldbte] bytes: 128 x 128 boxes, 128-byte swizzle
    if (!make_map(&mb, Bte, CU_TENSOR_MAP_DATA_TYPE_UINT8, D, K, ldbte, kBK, 128, CU_TENSOR_MAP_SWIZZLE_128B))
      return cudaErrorInvalidValue;
  } else if (!make_map(&mb, Sg, CU_TENSOR_MAP_DATA_TYPE_UINT32, lds, K, lds * 4, kCodesStageK / 32, 128,
                       CU_TENSOR_MAP_SWIZZLE_NONE)) {
    return cudaErrorInvalidValue;
  }
  TcArgs a{};
  const int khw = kh * kw, cb = 128 / khw;
  a.M = max_rows; a.N = K; a.L = D; a.count = count; a.rows_per_count = (int64_t)Ho * Wo;
  a.k_tiles = (int)((D + kCodesStageK - 1) / kCodesStageK); a.tiles_per_split = a.k_tiles;
  a.epi = EPI_FOLD; a.y = dx; a.kept_idx = kept_idx; a.scale = scale; a.zero = zero; a.cs = cs;
  a.rpg = (int64_t)Ho * Wo; a.status = status;
  a.n_step = cb * khw; a.grid_x = (C + cb - 1) / cb;
  a.fC = C; a.fH = H; a.fW = W; a.fkh = kh; a.fkw = kw; a.fstride = stride; a.fpad = pad; a.fHo = Ho; a.fWo = Wo;
  a.fcb = cb; a.fN = N; a.slot_of_group = slot_of_group;
  a.fd_khw = FastDiv((uint32_t)khw); a.fd_w = FastDiv((uint32_t)W); a.fd_kw = FastDiv((uint32_t)kw);
  a.fd_hw = FastDiv((uint32_t)(H * W)); a.fd_s = FastDiv((uint32_t)stride); a.fd_cbhw = FastDiv((uint32_t)(cb * H * W));
  // codes < 16 (b <= 4) go to the tensor cores straight from TMA (A_DIRECT)
  if (Bte) {  // the e4m3 B path writes NCHW only
    if (nhwc) return cudaErrorNotSupported;
    if (bits == 8) return launch_tc<true, true, 128, true, 2>(ma, mb, a, 1, s);
    return launch_tc<true, false, 128, true, 2 | 8>(ma, mb, a, 1, s);
  }
  if (nhwc) {
    if (bits == 8) return launch_tc<true, true, 128, true, 4>(ma, mb, a, 1, s);
    return launch_tc<true, false, 128, true, 4 | 8>(ma, mb, a, 1, s);
  }
  if (bits == 8) return launch_tc<true, true, 128, true>(ma, mb, a, 1, s);
  return launch_tc<true, false, 128, true, 8>(ma, mb, a, 1, s);
}

// Clusters of `cs` CTAs of this kernel that fit on the GPU at once (0 if unknown).
template <bool BITS8>
static int max_active_clusters(int cs) {
  using S = TcSmem<true, BITS8, 128>;
  // per device ordinal and cluster size: the number of clusters + 1 (0 = not yet known)
  static std::atomic<int> cache[64][9];
  static std::atomic<uint64_t> attr_bits{0};
  int dev = 0;
  if (cs < 1 || cs > 8 || cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  const int known = cache[dev][cs].load(std::memory_order_acquire);
  if (known > 0) return known - 1;
  auto kern = tc_gemm_kernel<true, BITS8, 128, false, BITS8 ? 0 : 8>;  // the kernel launch_wgrad_cluster_tc runs
  if (smem_attr_once((const void*)kern, S::kBytes, attr_bits) != cudaSuccess) return 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(1, 1, (unsigned)cs);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = S::kBytes;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 1;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = (unsigned)cs;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, (const void*)kern, &cfg) != cudaSuccess) {
    cudaGetLastError();
    n = 0;
  }
  cache[dev][cs].store(n + 1, std::memory_order_release);
  return n;
}

int wgrad_cluster_size(int bits, int64_t out_tiles, int64_t k_tiles) {
  // the largest cluster (<= 8 splits) whose out_tiles clusters all run in one wave
  for (int cs = 8; cs >= 1; --cs) {
    if (cs > k_tiles) continue;
    const int fit = bits == 8 ? max_active_clusters<true>(cs) : max_active_clusters<false>(cs);
    if (fit >= out_tiles) return cs;
  }
  return 1;
}

cudaError_t launch_wgrad_cluster_tc(int bits, const uint8_t* Q, int64_t ldq, int64_t capacity, const int32_t* count,
                                    const uint32_t* Sx, int64_t K, int64_t M, int splits, int32_t* acc, float* dw,
                                    int64_t D, const int32_t* kept_idx, const int32_t* slot_of_group,
                                    const float* scale, const float* zero, const int32_t* cs, int32_t* status,
                                    cudaStream_t s, const uint8_t* Be, int64_t ldbe) {
  const int64_t lds = fqt1_packed_words(M);
  CUtensorMap ma, mb;
  if (!make_map(&ma, Q, CU_TENSOR_MAP_DATA_TYPE_UINT8, M, capacity, ldq, kBK, kBM, CU_TENSOR_MAP_SWIZZLE_128B))
    return cudaErrorInvalidValue;
  if (Be) {  // e4m3 sign(X_u)^T rows [K][ldbe] bytes: 128 x 128 boxes, 128-byte swizzle
    if (!make_map(&mb, Be, CU_TENSOR_MAP_DATA_TYPE_UINT8, M, K, ldbe, kBK, 128, CU_TENSOR_MAP_SWIZZLE_128B))
      return cudaErrorInvalidValue;
  } else if (!make_map(&mb, Sx, CU_TENSOR_MAP_DATA_TYPE_UINT32, lds, K, lds * 4, kCodesStageK / 32, 128,
                       CU_TENSOR_MAP_SWIZZLE_NONE)) {
    return cudaErrorInvalidValue;
  }
  TcArgs a{};
  a.M = capacity; a.N = K; a.L = M; a.count = count; a.rows_per_count = 1;
  a.k_tiles = (int)((M + kCodesStageK - 1) / kCodesStageK);
  a.tiles_per_split = (a.k_tiles + splits - 1) / splits;
  a.epi = EPI_CRED; a.acc = acc; a.y = dw; a.ldo = K; a.kept_idx = kept_idx; a.scale = scale; a.zero = zero;
  a.cs = cs; a.status = status; a.slot_of_group = slot_of_group; a.D = D;
  if (Be) {
    if (bits == 8) return launch_tc<true, true, 128, false, 2>(ma, mb, a, splits, s, nullptr, nullptr, true);
    return launch_tc<true, false, 128, false, 2 | 8>(ma, mb, a, splits, s, nullptr, nullptr, true);
  }
  if (bits == 8) return launch_tc<true, true, 128>(ma, mb, a, splits, s, nullptr, nullptr, true);
  return launch_tc<true, false, 128, false, 8>(ma, mb, a, splits, s, nullptr, nullptr, true);
}

// grad_input product with its int32 accumulators column-major: acc[k * ld + r] for the kept
// rows r (EPI_ACC32 with acc_cm; ld >= max_rows).
cudaError_t launch_codes_tc_colmajor(int bits, const uint8_t* Q, int64_t ldq, int64_t max_rows, const int32_t* count,
                                     int64_t rows_per_count, const uint32_t* Sg, int64_t n_s, int64_t L,
                                     void* acc, int acc_bits, int64_t ld, int32_t* status, cudaStream_t s,
                                     const uint8_t* Be, int64_t ldbe) {
  TcArgs a{};
  a.acc = reinterpret_cast<int32_t*>(acc); a.ldo = ld; a.acc_cm = acc_bits == 16 ? 2 : 1;
  a.rpg = rows_per_count; a.status = status;
  return launch_codes_tc(bits, Q, ldq, max_rows, count, rows_per_count, Sg, n_s, L, EPI_ACC32, 1, a, s, Be, ldbe);
}

cudaError_t launch_codes_tc_simple(int bits, const uint8_t* Q, int64_t ldq, int64_t max_rows, const int32_t* count,
                                   int64_t rows_per_count, const uint32_t* Sg, int64_t n_s, int64_t L, int epi,
                                   int splits, int32_t* acc, float* out, int64_t ldo, const int32_t* kept_idx,
                                   const float* scale, const float* zero, const int32_t* cs, int64_t rpg,
                                   int32_t* status, cudaStream_t s, const uint8_t* Be, int64_t ldbe) {
  TcArgs a{};
  a.acc = acc; a.y = out; a.ldo = ldo; a.kept_idx = kept_idx; a.scale = scale; a.zero = zero; a.cs = cs;
  a.rpg = rpg; a.status = status;
  return launch_codes_tc(bits, Q, ldq, max_rows, count, rows_per_count, Sg, n_s, L, epi, splits, a, s, Be, ldbe);
}

}  // namespace fqt1
