// AGP + SCQ gradient quantization (Sec. 3.2, 5.2, 5.3).
//
//   range_kernel     one read of G = gY (.) gamma: per-sample-group and per-channel
//                    min / max through order-preserving integer atomics (exact).
//   select_kernel    one CTA per grouping: fixed-point ranges, water-filled keep
//                    probabilities, masks, kept list, scales S' and zero points Z'.
//   quantize_kernel  second read of G: stochastic rounding of the kept sample
//                    groups (PSQ codes, row-major) and kept channels (PCQ codes,
//                    written transposed through shared memory).
#include <algorithm>
#include <mutex>
#include <stdio.h>

#include "common.cuh"

namespace fqt1 {

// ------------------------------------------------------------------ ranges
constexpr int kRangeLoads = 4;  // float4 loads per thread per chunk

// Lane layout of the range pass: LPR lanes of 4 columns each span the CTA's column tile and a
// warp-wide load covers 32 / LPR rows.  The narrow layouts (LPR 16 or 8) keep every lane busy
// when D <= 64, where the full-width one would leave half or three quarters of them idle.
template <int LPR>
struct RangeShape {
  static constexpr int kRW = 32 / LPR;              // rows of one warp-wide load
  static constexpr int kChunk = kRangeLoads * kRW;  // rows of one warp per row tile
  static constexpr int kTile = 8 * kChunk;          // rows of one CTA per row tile
  static constexpr int kCols = 4 * LPR;             // columns of one CTA
};

struct RangeArgs {
  const float* g;
  const float* gamma;
  int64_t M, D, rpg;
  uint32_t *smin, *smax;  // [M / rpg] or null (smax holds complemented keys)
  uint32_t *cmin, *cmax;  // [D] or null (cmax holds complemented keys)
  int32_t* dev_status;
  FastDiv div_rpg;        // row -> sample group (rows < 2^31)
};

// Loads of a kernel's prologue are issued unconditionally, from a clamped index (or from
// `any`, a valid address, when the array is absent), and the result is selected afterwards:
// a load under a condition is not hoisted above the code before it, and a chain of them
// costs one memory round trip each.
template <class T>
__device__ __forceinline__ T ldg_sel(const T* p, int64_t i, bool ok, T dflt, const void* any) {
  const T v = __ldg(p ? p + (ok ? i : 0) : reinterpret_cast<const T*>(any));
  return ok ? v : dflt;
}

// One chunk of a lane: rows r, r + kRW, ... (clamped to the last row, so every address is valid)
// and columns c0 .. c0 + 3 (clamped likewise; the caller masks what lies outside G).
template <int LPR, bool VEC>
__device__ __forceinline__ void range_load(const RangeArgs& a, int64_t r, int64_t c0, bool cv0,
                                           float (&v)[kRangeLoads][4]) {
#pragma unroll
  for (int i = 0; i < kRangeLoads; ++i) {
    const int64_t ri = min(r + i * RangeShape<LPR>::kRW, a.M - 1);
    if (VEC) {
      const float4 t = __ldg(reinterpret_cast<const float4*>(a.g + ri * a.D + (cv0 ? c0 : 0)));
      v[i][0] = t.x; v[i][1] = t.y; v[i][2] = t.z; v[i][3] = t.w;
    } else {
#pragma unroll
      for (int q = 0; q < 4; ++q) v[i][q] = __ldg(a.g + ri * a.D + min(c0 + q, a.D - 1));
    }
  }
}

// The range pass is bound by instructions and load latency per element, not by memory, so its
// loop is lean: float minima / maxima per thread (ordered integer keys only for the atomics),
// one finite test per element, the Gamma product only when there is a Gamma (the loop exists
// in both forms), and the sample-group bookkeeping once per chunk of a warp when the chunk lies
// in one group (the usual case: a group is a whole sample).  rc is the chunk's first row
// (warp-uniform), sub the lane's row within a warp-wide load.
template <int LPR, bool GAMMA>
__device__ __forceinline__ void range_chunk(const RangeArgs& a, int64_t rc, int sub, const bool (&cv)[4],
                                            const float (&gam)[4], const float (&v)[kRangeLoads][4],
                                            float (&cmn)[4], float (&cmx)[4], float& gmn, float& gmx,
                                            int64_t& cur, bool& bad, int lane) {
  using S = RangeShape<LPR>;
  const int nrows = (int)min((int64_t)S::kChunk, a.M - rc);  // >= 1
  const int64_t g0 = a.div_rpg.div((uint32_t)rc), g1 = a.div_rpg.div((uint32_t)(rc + nrows - 1));
  auto flush = [&](int64_t next) {  // the warp's group minimum / maximum, when its rows move on
    if (a.smin && next != cur) {
      if (cur >= 0) {
        const uint32_t mn = __reduce_min_sync(0xFFFFFFFFu, float_to_ordered(gmn));
        const uint32_t mx = __reduce_max_sync(0xFFFFFFFFu, float_to_ordered(gmx));
        if (lane == 0) { atomicMin(a.smin + cur, mn); atomicMin(a.smax + cur, ~mx); }
      }
      cur = next;
      gmn = __int_as_float(0x7F800000);   // +inf
      gmx = __int_as_float(0xFF800000);   // -inf
    }
  };
  auto take = [&](float g, int q) {
    const float x = GAMMA ? __fmul_rn(g, gam[q]) : g;
    bad |= !(fabsf(x) <= 3.402823466e38f);  // NaN or +-Inf
    cmn[q] = fminf(cmn[q], x); cmx[q] = fmaxf(cmx[q], x);
    return x;
  };
  if (g0 == g1) {
    flush(g0);
#pragma unroll
    for (int i = 0; i < kRangeLoads; ++i) {
      const bool rv = i * S::kRW + sub < nrows;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        if (!cv[q] || !rv) continue;
        const float x = take(v[i][q], q);
        gmn = fminf(gmn, x); gmx = fmaxf(gmx, x);
      }
    }
  } else if (LPR == 32) {  // one row per load: the warp follows the group boundary row by row
    int64_t gi = g0, grem = rc - g0 * a.rpg;
#pragma unroll
    for (int i = 0; i < kRangeLoads; ++i) {
      if (i >= nrows) break;
      if (i > 0 && ++grem == a.rpg) { grem = 0; ++gi; }
      flush(gi);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        if (!cv[q]) continue;
        const float x = take(v[i][q], q);
        gmn = fminf(gmn, x); gmx = fmaxf(gmx, x);
      }
    }
  } else {  // lanes of one load in different groups (the host avoids this layout then): per element
    flush(-1);
#pragma unroll
    for (int i = 0; i < kRangeLoads; ++i) {
      if (i * S::kRW + sub >= nrows) continue;
      const int64_t gi = a.div_rpg.div((uint32_t)(rc + i * S::kRW + sub));
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        if (!cv[q]) continue;
        const float x = take(v[i][q], q);
        if (a.smin) { atomicMin(a.smin + gi, float_to_ordered(x)); atomicMin(a.smax + gi, ~float_to_ordered(x)); }
      }
    }
  }
}

// A contiguous run of row tiles per CTA: the host sizes gridDim.y to one resident wave, so that a
// tall gradient (the ResNet-18 stem: 12544 row tiles) updates each channel key once per CTA
// rather than once per row tile, and a warp's rows leave a sample group at most a few times
// (strided tiles would change group on every tile and flood the group keys with atomics).  The
// next chunk's loads are issued before the current chunk is reduced, so that every lane keeps
// two chunks of G in flight.
template <int LPR, bool VEC>
__global__ void __launch_bounds__(256) range_kernel(RangeArgs a) {
  using S = RangeShape<LPR>;
  FQT1_PDL_WAIT();
  FQT1_PDL_TRIGGER();
  __shared__ uint32_t cmin_s[8][S::kCols], cmax_s[8][S::kCols];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, sub = lane / LPR;
  const int64_t c0 = (int64_t)blockIdx.x * S::kCols + (lane % LPR) * 4;
  float gam[4];
  bool cv[4];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    cv[q] = c0 + q < a.D;
    gam[q] = ldg_sel(a.gamma, c0 + q, a.gamma && cv[q], 1.0f, a.g);
  }
  const float pinf = __int_as_float(0x7F800000), ninf = __int_as_float(0xFF800000);
  float cmn[4] = {pinf, pinf, pinf, pinf}, cmx[4] = {ninf, ninf, ninf, ninf};
  float gmn = pinf, gmx = ninf;
  int64_t cur = -1;
  bool bad = false;
  const int64_t row_tiles = (a.M + S::kTile - 1) / S::kTile;
  const int64_t per_cta = (row_tiles + gridDim.y - 1) / gridDim.y;
  const int64_t rt0 = (int64_t)blockIdx.y * per_cta, rt1 = min(row_tiles, rt0 + per_cta);
  const int64_t wrow = (int64_t)warp * S::kChunk;
  float v[kRangeLoads][4], nv[kRangeLoads][4];
  if (rt0 < rt1) range_load<LPR, VEC>(a, rt0 * S::kTile + wrow + sub, c0, cv[0], v);
#pragma unroll 1
  for (int64_t rt = rt0; rt < rt1; ++rt) {
    const int64_t rc = rt * S::kTile + wrow;
    if (rc >= a.M) break;  // warp-uniform; later tiles start further on
    if (rt + 1 < rt1) range_load<LPR, VEC>(a, rc + S::kTile + sub, c0, cv[0], nv);
    if (a.gamma) range_chunk<LPR, true>(a, rc, sub, cv, gam, v, cmn, cmx, gmn, gmx, cur, bad, lane);
    else range_chunk<LPR, false>(a, rc, sub, cv, gam, v, cmn, cmx, gmn, gmx, cur, bad, lane);
#pragma unroll
    for (int i = 0; i < kRangeLoads; ++i)
#pragma unroll
      for (int q = 0; q < 4; ++q) v[i][q] = nv[i][q];
  }
  // rc is warp-uniform, so every lane of a warp that has rows reaches this flush together
  if (a.smin && cur >= 0) {
    const uint32_t mn = __reduce_min_sync(0xFFFFFFFFu, float_to_ordered(gmn));
    const uint32_t mx = __reduce_max_sync(0xFFFFFFFFu, float_to_ordered(gmx));
    if (lane == 0) { atomicMin(a.smin + cur, mn); atomicMin(a.smax + cur, ~mx); }
  }
  if (__any_sync(0xFFFFFFFFu, bad) && lane == 0) atomicOr(a.dev_status, FQT1_DEV_NONFINITE);
  if (a.cmin) {
#pragma unroll
    for (int q = 0; q < 4; ++q) {  // lanes that hold the same columns (other rows) first
#pragma unroll
      for (int o = LPR; o < 32; o <<= 1) {
        cmn[q] = fminf(cmn[q], __shfl_xor_sync(0xFFFFFFFFu, cmn[q], o));
        cmx[q] = fmaxf(cmx[q], __shfl_xor_sync(0xFFFFFFFFu, cmx[q], o));
      }
    }
    if (lane < LPR) {
#pragma unroll
      for (int q = 0; q < 4; ++q) {  // no rows: +inf / -inf map to keys that leave the atomics below idle
        cmin_s[warp][lane * 4 + q] = float_to_ordered(cmn[q]);
        cmax_s[warp][lane * 4 + q] = cmx[q] == ninf ? 0u : float_to_ordered(cmx[q]);
      }
    }
    __syncthreads();
    if (threadIdx.x < S::kCols) {
      const int64_t c = (int64_t)blockIdx.x * S::kCols + threadIdx.x;
      uint32_t mn = 0xFFFFFFFFu, mx = 0u;
#pragma unroll
      for (int w = 0; w < 8; ++w) { mn = min(mn, cmin_s[w][threadIdx.x]); mx = max(mx, cmax_s[w][threadIdx.x]); }
      if (c < a.D && mx != 0u) { atomicMin(a.cmin + c, mn); atomicMin(a.cmax + c, ~mx); }
    }
  }
}

// --------------------------------------------------------------- selection
struct SelectArgs {
  uint32_t* kmin;  // the range keys of the grouping; reset to 0xFFFFFFFF once read
  uint32_t* kmax;
  int32_t n, bits, mode, capacity;
  uint64_t seed;
  uint32_t stream;
  fqt1_qgrad out;
};

constexpr int kSelThreads = 1024;

// Inclusive scan of one uint64 per thread across the CTA's NT threads; returns the inclusive
// value and writes the CTA total to *total.
template <int NT>
__device__ uint64_t block_inclusive_scan(uint64_t v, uint64_t* warp_sums, uint64_t* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint64_t t = __shfl_up_sync(0xFFFFFFFFu, v, o);
    if (lane >= o) v += t;
  }
  if (lane == 31) warp_sums[warp] = v;
  __syncthreads();
  if (warp == 0) {
    uint64_t s = lane < NT / 32 ? warp_sums[lane] : 0ull;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint64_t t = __shfl_up_sync(0xFFFFFFFFu, s, o);
      if (lane >= o) s += t;
    }
    warp_sums[lane] = s;
  }
  __syncthreads();
  if (warp > 0) v += warp_sums[warp - 1];
  const uint64_t tot = warp_sums[31];
  __syncthreads();
  *total = tot;
  return v;
}

// floor(a * 2^32 / d) for 0 < d < 2^62, a < 2^60 (exact; quotients of 2^34 or more return ~0,
// the callers clamp at 2^32).  An fp32 estimate (relative error below 2^-20) is corrected with
// exact 128-bit remainders; float64 is avoided (its division is slow on this part).  The float
// quotients are the fast approximate ones: the integer steps after them make the result exact.
__device__ __forceinline__ uint64_t div_shift32(uint64_t a, uint64_t d) {
  typedef unsigned __int128 u128;
  const u128 num = (u128)a << 32;
  if ((num >> 34) >= d) return ~0ull;
  uint64_t q = (uint64_t)__fdividef(__ull2float_rn(a), __fmul_rn(__ull2float_rn(d), 2.3283064365386963e-10f));
  // |q - quotient| < 2^15: one float step on the remainder, scaled so that d keeps 24 bits
  const int sh = max(0, 40 - __clzll(d));
  const float df = __ull2float_rn(d >> sh);
  const u128 qd = (u128)q * d;
  if (qd > num) q -= (uint64_t)__fdividef(__ull2float_rn((uint64_t)((qd - num) >> sh)), df);
  else q += (uint64_t)__fdividef(__ull2float_rn((uint64_t)((num - qd) >> sh)), df);
  while ((u128)q * d > num) --q;
  while ((u128)(q + 1) * d <= num) ++q;
  return q;
}

// p^ = P 2^-32 as a float64, built from its bits (P <= 2^33).
__device__ __forceinline__ double p_hat_of(uint64_t P) {
  if (P == 0) return 0.0;
  const int lz = __clzll(P);
  const uint64_t frac = ((P << lz) << 1) >> 12;  // fraction bits below the leading one
  const uint64_t ex = (uint64_t)(1023 + 63 - lz - 32);
  return __longlong_as_double((long long)((ex << 52) | frac));
}

// NT threads per CTA (256 when every grouping has at most 256 groups, else 1024).
template <int NT>
__global__ void __launch_bounds__(NT) select_kernel(SelectArgs a0, SelectArgs a1) {
  // The dependents (the quantize grid, one CTA per tile of G) are released only when this
  // kernel ends: launched early they would occupy every SM in their dependency wait while
  // these two CTAs run, keeping the other branches' kernels off the GPU.
  FQT1_PDL_WAIT();
  const SelectArgs& a = blockIdx.x == 0 ? a0 : a1;
  extern __shared__ __align__(16) unsigned char sel_smem[];
  __shared__ uint64_t warp_sums[32];
  __shared__ uint32_t s_rmax;
  __shared__ int s_tstar;
  __shared__ uint64_t s_kth, s_stot;
  __shared__ int rank_s[NT];
  __shared__ uint64_t sorted_s[NT];
  const int n = a.n, tid = threadIdx.x;
  if (n <= 0) return;
  int npad = 1;
  while (npad < n) npad <<= 1;
  uint64_t* key = reinterpret_cast<uint64_t*>(sel_smem);           // [npad] sort keys, later P
  float* rf = reinterpret_cast<float*>(sel_smem + 8 * (size_t)npad);  // [n] ranges
  const fqt1_qgrad& o = a.out;

  // Z = min, R = max - min (fp32)
  if (tid == 0) s_rmax = 0u;
  __syncthreads();
  for (int i = tid; i < n; i += NT) {
    const float z = ordered_to_float(a.kmin[i]);
    const float r = __fsub_rn(ordered_to_float(~a.kmax[i]), z);
    // the keys go back to their initial value for the next call's range pass (the only other
    // reader of them, which runs before this kernel), so no call needs to fill them first
    a.kmin[i] = 0xFFFFFFFFu;
    a.kmax[i] = 0xFFFFFFFFu;
    o.group_min[i] = z;
    o.group_range[i] = r;
    rf[i] = r;
    if (r > 0.0f) atomicMax(&s_rmax, __float_as_uint(r));
  }
  __syncthreads();
  const float rmax = __uint_as_float(s_rmax);
  const uint64_t two32 = 1ull << 32;

  // Fixed-point ranges R~ = floor(R 2^(40 - E)), 2^(E-1) <= max R < 2^E.
  int e = 0;
  if (rmax > 0.0f) frexpf(rmax, &e);
  // R~ = floor(R 2^(40 - E)) from the bits of R = m 2^x (exact integer shifts)
  auto rtilde = [&](int i) -> uint64_t {
    const float r = rf[i];
    if (!(rmax > 0.0f) || !(r > 0.0f)) return 0ull;
    const uint32_t b = __float_as_uint(r);
    const int eb = (int)((b >> 23) & 0xFFu);
    const uint64_t m = eb ? ((b & 0x7FFFFFu) | 0x800000u) : (b & 0x7FFFFFu);
    const int sh = min((eb ? eb - 150 : -149) + kFixedPointBits - e, kFixedPointBits);
    return sh >= 0 ? (m << sh) : (sh <= -32 ? 0ull : (m >> -sh));
  };

  if (a.bits > 1 && n <= NT) {
    // rank of each key (R~ desc, index asc) by comparison with all others: no sort needed
    uint64_t myk = 0, myrt = 0;
    if (tid < n) {
      myrt = rtilde(tid);
      myk = (myrt << 24) | (uint64_t)(0xFFFFFFu - (uint32_t)tid);
      key[tid] = myk;
    }
    // rank of each key: every warp sorts its 32 keys (bitonic, shuffles), then a key's rank is
    // the number of larger keys in all the sorted lists (a 5-step binary search in each)
    {
      const int lane = tid & 31, nw = (n + 31) >> 5;
      if ((tid >> 5) < nw) {
        uint64_t k = tid < n ? myk : 0ull;
#pragma unroll
        for (int size = 2; size <= 32; size <<= 1) {
#pragma unroll
          for (int stride = size >> 1; stride > 0; stride >>= 1) {
            const uint64_t o = __shfl_xor_sync(0xFFFFFFFFu, k, stride);
            const bool take_max = ((lane & stride) == 0) == ((lane & size) == 0);
            k = take_max ? (k > o ? k : o) : (k < o ? k : o);
          }
        }
        sorted_s[tid] = k;
      }
      __syncthreads();
      if (tid < n) {
        int r = 0;
        for (int w = 0; w < nw; ++w) {
          const uint64_t* L = sorted_s + 32 * w;
          int idx = 0;
#pragma unroll
          for (int step = 16; step >= 1; step >>= 1)
            if (L[idx + step - 1] > myk) idx += step;
          if (idx == 31 && L[31] > myk) idx = 32;  // the five steps reach at most 31
          r += idx;
        }
        rank_s[tid] = r;
      }
    }
    __syncthreads();
    const int rank = tid < n ? rank_s[tid] : 0;
    if (tid < n) key[rank] = myrt;  // fixed-point ranges in sorted (descending) order
    __syncthreads();
    int tstar;
    uint64_t S = 0;
    if (a.mode == FQT1_SEL_TOPK) {
      tstar = max(1, n / a.bits);
    } else {
      // thread u holds position t = n - 1 - u; its inclusive scan is the suffix sum S_t
      const int t = n - 1 - tid;
      const uint64_t v = (tid < n) ? key[t] : 0ull;
      uint64_t total;
      const uint64_t suffix = block_inclusive_scan<NT>(v, warp_sums, &total);
      if (tid == 0) s_tstar = n;
      __syncthreads();
      if (tid < n) {
        const int64_t lhs = (int64_t)(n - a.bits * t) * (int64_t)v;
        if (lhs <= (int64_t)a.bits * (int64_t)suffix) atomicMin(&s_tstar, t);
      }
      __syncthreads();
      tstar = s_tstar;
      if (tid < n && t == tstar) s_stot = suffix;
      if (tid == 0 && tstar >= n) s_stot = 0;
      __syncthreads();
      S = s_stot;
    }
    __syncthreads();
    if (tid < n) {
      uint64_t P;
      if (a.mode == FQT1_SEL_TOPK) P = rank < tstar ? two32 : 0ull;
      else if (rank < tstar) P = two32;
      else if (S > 0) P = min(two32, div_shift32((uint64_t)(n - a.bits * tstar) * myrt, (uint64_t)a.bits * S));
      else P = 0;
      key[tid] = P;
    }
  } else if (a.bits > 1) {
    // sort keys (R~ desc, index asc) descending
    for (int i = tid; i < npad; i += NT)
      key[i] = i < n ? ((rtilde(i) << 24) | (uint64_t)(0xFFFFFFu - (uint32_t)i)) : 0ull;
    __syncthreads();
    for (int size = 2; size <= npad; size <<= 1) {
      for (int stride = size >> 1; stride > 0; stride >>= 1) {
        for (int i = tid; i < npad / 2; i += NT) {
          const int lo = 2 * i - (i & (stride - 1));
          const int hi = lo + stride;
          const bool desc = (lo & size) == 0;
          const uint64_t x = key[lo], y = key[hi];
          if ((x < y) == desc) { key[lo] = y; key[hi] = x; }
        }
        __syncthreads();
      }
    }
    if (a.mode == FQT1_SEL_TOPK) {
      const int k = max(1, n / a.bits);
      if (tid == 0) { s_kth = key[k - 1]; s_tstar = k; s_stot = 0; }
    } else {
      // suffix sums S_t over sorted positions; t* = first t with (n - b t) R~_(t) <= b S_t
      const int per = (npad + NT - 1) / NT;
      const int beg = min(npad, tid * per), end = min(npad, beg + per);
      uint64_t local = 0;
      for (int t = beg; t < end; ++t) local += key[t] >> 24;
      // suffix of thread chunks: scan reversed thread order
      uint64_t total;
      const uint64_t incl = block_inclusive_scan<NT>(local, warp_sums, &total);
      uint64_t suffix = total - incl + local;  // sum of positions >= beg
      int best = n;
      uint64_t best_s = 0;
      for (int t = beg; t < end && t < n; ++t) {
        const uint64_t rt = key[t] >> 24;
        const int64_t lhs = (int64_t)(n - a.bits * t) * (int64_t)rt;
        const int64_t rhs = (int64_t)a.bits * (int64_t)suffix;
        if (lhs <= rhs) { best = t; best_s = suffix; break; }
        suffix -= rt;
      }
      if (tid == 0) s_tstar = n;
      __syncthreads();
      atomicMin(&s_tstar, best);
      __syncthreads();
      if (best == s_tstar && best < n) { s_stot = best_s; s_kth = key[best]; }
      if (tid == 0 && s_tstar >= n) { s_stot = 0; s_kth = 0; }
    }
    __syncthreads();
    // P_i by group index (reuses the key buffer)
    const int tstar = s_tstar;
    const uint64_t kth = s_kth, S = s_stot;
    for (int i = tid; i < n; i += NT) {
      const uint64_t rt = rtilde(i);
      const uint64_t ki = (rt << 24) | (uint64_t)(0xFFFFFFu - (uint32_t)i);
      uint64_t P;
      if (a.mode == FQT1_SEL_TOPK) {
        P = ki >= kth ? two32 : 0ull;
      } else if (ki > kth) {
        P = two32;
      } else if (S > 0) {
        const uint64_t num = (uint64_t)(n - a.bits * tstar) * rt;
        P = min(two32, div_shift32(num, (uint64_t)a.bits * S));
      } else {
        P = 0;
      }
      key[i] = P;
    }
  } else {
    for (int i = tid; i < n; i += NT) key[i] = two32;
  }
  __syncthreads();

  // masks in index order; each thread owns a contiguous chunk
  const int per = (n + NT - 1) / NT;
  const int beg = min(n, tid * per), end = min(n, beg + per);
  uint64_t psum = 0;
  for (int i = beg; i < end; ++i) psum += key[i];
  uint64_t total;
  const uint64_t pincl = block_inclusive_scan<NT>(psum, warp_sums, &total);
  uint64_t c = pincl - psum;
  uint64_t u = 0;
  if (a.bits > 1 && a.mode == FQT1_SEL_SYSTEMATIC) u = philox_word(a.seed, a.stream, 0);
  c += u;
  uint64_t kept_bits = 0;  // chunk length <= 64 for n <= 16384 and NT >= 256
  int nk = 0;
  for (int i = beg; i < end; ++i) {
    const uint64_t P = key[i];
    bool kept;
    if (a.bits == 1) kept = true;
    else if (a.mode == FQT1_SEL_SYSTEMATIC) kept = ((c + P) >> 32) > (c >> 32);
    else if (a.mode == FQT1_SEL_BERNOULLI) kept = (uint64_t)philox_word(a.seed, a.stream, (uint64_t)i) < P;
    else kept = P == two32;
    c += P;
    if (kept) { kept_bits |= 1ull << (i - beg); ++nk; }
  }
  uint64_t ktot;
  const uint64_t kincl = block_inclusive_scan<NT>((uint64_t)nk, warp_sums, &ktot);
  int slot = (int)(kincl - nk);
  // Finite gradients never keep more than `capacity` groups (systematic: floor or ceil of
  // sum p^ <= n / b; top-k: n / b; Bernoulli and b = 1: capacity = n).  A non-finite range
  // (flagged by the range pass) breaks the fixed-point arithmetic above, so the kept list is
  // cut at the capacity here: no later kernel reads or writes past the caller's buffers.
  const int kcap = (int)min(ktot, (uint64_t)a.capacity);
  // the per-slot scale and zero point are computed by the quantize kernel
  for (int i = beg; i < end; ++i) {
    const uint64_t P = key[i];
    o.p_hat[i] = p_hat_of(P);
    if ((kept_bits & (1ull << (i - beg))) && slot < kcap) {
      o.slot_of_group[i] = slot;
      o.kept_idx[slot] = i;
      ++slot;
    } else {
      o.slot_of_group[i] = -1;
    }
  }
  for (int s = kcap + tid; s < a.capacity; s += NT) o.kept_idx[s] = -1;
  if (tid == 0) *o.kept_count = (int32_t)kcap;
}

// --------------------------------------------------------------- quantize
struct QBranch {
  const float* zmin;     // [n] group minima
  const float* range;    // [n] group ranges
  const int32_t* slot;   // [n] slot or -1
  uint8_t* codes;
  int64_t ld;
  float B;
  uint64_t seed;
  const int32_t* kept_idx;    // [capacity] group of each slot
  const int32_t* kept_count;  // [1]
  const double* p_hat;        // [n]
  float* scale;               // [capacity] S' = R / (B p^)
  float* zero;                // [capacity] Z' = Z / p^
};

constexpr int kQWarps = 8;  // quantizing warps; one more warp computes the per-slot constants

// Dequantization constants of the kept slots (Sec. 5.3): S' = R / (B p^) and Z' = Z / p^ in
// float64, rounded to float, for slots cta, cta + ncta, ...  Lanes 0 / 1 compute the sample
// branch's S' / Z', lanes 2 / 3 the channel branch's, all four in the same instructions.
__device__ void slot_constants(const QBranch& bs, const QBranch& bc, bool do_s, bool do_c, int64_t cta,
                               int64_t ncta, int lane) {
  const bool chan = lane >= 2, zero_pt = (lane & 1) != 0;
  if (lane >= 4 || !(chan ? do_c : do_s)) return;
  const QBranch& q = chan ? bc : bs;
  const int32_t count = __ldg(q.kept_count);
  for (int64_t s = cta; s < count; s += ncta) {
    const int32_t i = __ldg(q.kept_idx + s);
    const double ph = __ldg(q.p_hat + i);
    const double num = (double)__ldg((zero_pt ? q.zmin : q.range) + i);
    const double den = zero_pt ? ph : __dmul_rn((double)q.B, ph);
    (zero_pt ? q.zero : q.scale)[s] = __double2float_rn(__ddiv_rn(num, den));
  }
}

struct QuantArgs {
  const float* g;
  const float* gamma;
  int64_t M, D, rpg;
  int do_psq, do_pcq;
  QBranch s, c;
  FastDiv div_rpg;  // row -> sample group (rows < 2^31)
};

// Tile shape of the quantize pass: LPC lanes of 4 columns span kCols columns of G, a warp-wide
// load covers kRW = 32 / LPC rows, and each quantizing thread holds 4 x 4 values of a tile
// (kRows x kCols = 4096 elements for every LPC).  The narrow shapes (LPC 16 or 8) keep every
// lane busy when D <= 64, where the full-width one would leave half or three quarters idle.
template <int LPC>
struct QShape {
  static constexpr int kCols = 4 * LPC;
  static constexpr int kRW = 32 / LPC;       // rows of one warp-wide load
  static constexpr int kWarpRows = 4 * kRW;  // rows of one warp per tile
  static constexpr int kRows = kQWarps * kWarpRows;
};

// The values one lane holds for one tile: rows rw + kRW i (i < 4), columns c0 .. c0 + 3.
struct QRows {
  float v[4][4];
};

// Every load of a lane's tile, unconditional (clamped rows and columns), so that all of them
// are in flight together.
template <bool VEC, int RW>
__device__ __forceinline__ void quant_load(const QuantArgs& a, int64_t rw, int64_t c0, bool cv0, QRows& t) {
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int64_t rc = min(rw + (int64_t)i * RW, a.M - 1);
    if (VEC) {
      const float4 x = __ldg(reinterpret_cast<const float4*>(a.g + rc * a.D + (cv0 ? c0 : 0)));
      t.v[i][0] = x.x; t.v[i][1] = x.y; t.v[i][2] = x.z; t.v[i][3] = x.w;
    } else {
#pragma unroll
      for (int q = 0; q < 4; ++q) t.v[i][q] = __ldg(a.g + rc * a.D + min(c0 + q, a.D - 1));
    }
  }
}

// The sample-branch constants of a lane's rows rw + RW i: slot (-1: pruned, or past M), row in
// its group, range and zero point.  The loads are issued together and hit L1 / L2.
template <int RW>
__device__ __forceinline__ void quant_rows(const QuantArgs& a, int64_t rw, int32_t (&slot)[4], int32_t (&rem)[4],
                                           float (&rg)[4], float (&zm)[4]) {
  // one division for the first row; the next rows step by RW (at most one group boundary per
  // step when rpg >= RW, else a division each)
  const uint32_t r0 = (uint32_t)min(rw, a.M - 1);
  uint32_t gi = a.div_rpg.div(r0), rr = r0 - gi * (uint32_t)a.rpg;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int64_t r = rw + (int64_t)i * RW;
    if (i > 0) {
      if (a.rpg >= RW) {
        rr += RW;
        if (rr >= (uint32_t)a.rpg) { rr -= (uint32_t)a.rpg; ++gi; }
      } else {
        const uint32_t rc = (uint32_t)min(r, a.M - 1);
        gi = a.div_rpg.div(rc);
        rr = rc - gi * (uint32_t)a.rpg;
      }
    }
    rem[i] = (int32_t)rr;
    const bool ls = r < a.M;
    slot[i] = ldg_sel(a.s.slot, (int64_t)gi, ls, -1, a.g);
    rg[i] = ldg_sel(a.s.range, (int64_t)gi, ls, 0.f, a.g);
    zm[i] = ldg_sel(a.s.zmin, (int64_t)gi, ls, 0.f, a.g);
  }
}

// Codes of the tiles of G = gY * gamma for both branches (Sec. 5.3).
//  - Warps 0-7 quantize.  A CTA takes one column tile and every gridDim.y-th row tile (the
//    host sizes the grid to about one resident wave), and issues the next tile's loads before
//    it rounds the current one, so that every lane keeps two tiles of G in flight.
//  - PSQ: rows of kept sample groups; element (m, j) takes word m D + j of stream 0, so one
//    Philox block gives a lane's 4 columns of a row.
//  - PCQ: the tile goes to shared memory; one thread per (kept column, 4 rows) draws one
//    Philox block (words j M + m .. + 3 of stream 1) and forms the 4 codes, so no rounding is
//    spent on pruned channels.  The codes are staged in shared memory and written with the
//    samples contiguous.
//  - Warp 8 lists the kept columns of the column tile with their constants once (the list is
//    the same for every row tile), signals barrier 1 without waiting, then computes the
//    per-slot S' and Z' in float64 beside the quantizing warps.
//  - PIPE (row tiles beyond one resident wave): the next tile's loads are issued before the
//    current tile is rounded; the extra registers leave two CTAs per SM.  Without it a CTA
//    takes one tile at a time and four CTAs fit on an SM.
template <int LPC, bool VEC, bool PIPE>
__global__ void __launch_bounds__(32 * (kQWarps + 1), PIPE ? 2 : 4) quantize_kernel(QuantArgs a) {
  using S = QShape<LPC>;
  // the dependent (the grad_input product, a leaf of the step) is not released early either:
  // its CTAs would wait on SMs that the grad_weight product, which also waits for this
  // kernel, can use
  FQT1_PDL_WAIT();
  __shared__ __align__(16) float gt[S::kRows][S::kCols + 4];  // the tile of G * gamma
  __shared__ uint32_t tile[S::kCols][S::kRows / 4 + 1];       // codes of kept column j, 4 rows per word
  __shared__ int32_t klist[S::kCols], kslot[S::kCols];        // kept column j: tile column, slot
  __shared__ float kz[S::kCols], kinv[S::kCols];              // its Z and B / R (negative: degenerate)
  __shared__ int32_t nk_s;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t cb = (int64_t)blockIdx.x * S::kCols;
  if (warp == kQWarps) {
    if (a.do_pcq) {
      // the kept columns of the tile in ascending order (lane l: tile columns 4l .. 4l+3)
      const int64_t c0 = cb + lane * 4;
      int32_t cslot[4];
      float crg[4], zc[4];
      int mine = 0;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const bool lc = 4 * lane + q < S::kCols && c0 + q < a.D;
        cslot[q] = ldg_sel(a.c.slot, c0 + q, lc, -1, a.g);
        crg[q] = ldg_sel(a.c.range, c0 + q, lc, 0.f, a.g);
        zc[q] = ldg_sel(a.c.zmin, c0 + q, lc, 0.f, a.g);
      }
#pragma unroll
      for (int q = 0; q < 4; ++q) mine += cslot[q] >= 0 ? 1 : 0;
      int incl = mine;
#pragma unroll
      for (int d = 1; d < 32; d <<= 1) {
        const int t = __shfl_up_sync(0xFFFFFFFFu, incl, d);
        if (lane >= d) incl += t;
      }
      int j = incl - mine;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        if (cslot[q] < 0) continue;
        const float inv = __fdiv_rn(a.c.B, crg[q]);
        klist[j] = 4 * lane + q;
        kslot[j] = cslot[q];
        kz[j] = zc[q];
        kinv[j] = (!(crg[q] > 0.0f) || !isfinite(inv)) ? -1.0f : inv;
        ++j;
      }
      if (lane == 31) nk_s = incl;
      asm volatile("bar.arrive 1, %0;" ::"n"(32 * (kQWarps + 1)) : "memory");
    }
    // the float64 divisions run beside the quantizing warps of this CTA
    const int64_t cta = (int64_t)blockIdx.y * gridDim.x + blockIdx.x, ncta = (int64_t)gridDim.x * gridDim.y;
    slot_constants(a.s, a.c, a.do_psq != 0, a.do_pcq != 0, cta, ncta, lane);
    return;
  }
  const int sub = lane / LPC;
  const int64_t c0 = cb + (lane % LPC) * 4;
  float gam[4];
  bool cv[4];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int64_t c = c0 + q;
    cv[q] = c < a.D;
    gam[q] = ldg_sel(a.gamma, c, a.gamma && cv[q], 1.0f, a.g);
  }
  // row tiles blockIdx.y, + gridDim.y, ...: strided, so that every CTA gets its share of the
  // kept sample groups (their PSQ rounding costs several times a pruned tile's work)
  const int64_t row_tiles = (a.M + S::kRows - 1) / S::kRows;
  const int64_t rt0 = blockIdx.y, rstep = gridDim.y;
  const int64_t lrow = (int64_t)warp * S::kWarpRows + sub;  // this lane's first row in a tile
  // without PIPE the host launches one CTA per row tile, and the tile is not a loop
  QRows cur, nxt;
  auto do_tile = [&](int64_t rt) {
    const int64_t r0 = rt * S::kRows, rw = r0 + lrow;
    int32_t sslot[4], srem[4];
    float srg[4], szm[4];
    if (a.do_psq) quant_rows<S::kRW>(a, rw, sslot, srem, srg, szm);
    if (PIPE && rt + rstep < row_tiles) quant_load<VEC, S::kRW>(a, rw + rstep * S::kRows, c0, cv[0], nxt);
    if (a.gamma) {
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int q = 0; q < 4; ++q) cur.v[i][q] = __fmul_rn(cur.v[i][q], gam[q]);
    }
    // PSQ: kept rows; element (m, j) takes word m*D + j of stream 0 (one block = 4 columns)
#pragma unroll
    for (int i = 0; i < 4 && a.do_psq; ++i) {
      if (sslot[i] < 0) continue;
      const int64_t r = rw + (int64_t)i * S::kRW;
      const float rs = srg[i], zs = szm[i];
      const float inv = __fdiv_rn(a.s.B, rs);
      const bool deg = !(rs > 0.0f) || !isfinite(inv);
      const uint64_t e0 = (uint64_t)r * (uint64_t)a.D + (uint64_t)c0;
      uint8_t* dst = a.s.codes + ((int64_t)sslot[i] * a.rpg + srem[i]) * a.s.ld + c0;
      if (VEC) {
        if (cv[0]) {
          const U32x4 p = philox_block(a.s.seed, kStreamSrPsq, e0 >> 2);
          const uint32_t packed = sr_code(cur.v[i][0], zs, inv, a.s.B, deg, p.x) |
                                  (sr_code(cur.v[i][1], zs, inv, a.s.B, deg, p.y) << 8) |
                                  (sr_code(cur.v[i][2], zs, inv, a.s.B, deg, p.z) << 16) |
                                  (sr_code(cur.v[i][3], zs, inv, a.s.B, deg, p.w) << 24);
          *reinterpret_cast<uint32_t*>(dst) = packed;
        }
      } else {
#pragma unroll
        for (int q = 0; q < 4; ++q)
          if (cv[q])
            dst[q] = (uint8_t)sr_code(cur.v[i][q], zs, inv, a.s.B, deg, philox_word(a.s.seed, kStreamSrPsq, e0 + q));
      }
    }
    if (a.do_pcq) {
      // stage the tile; on the first tile barrier 1 also waits for warp 8's list of kept
      // columns, later tiles need only the quantizing warps (barrier 3)
#pragma unroll
      for (int i = 0; i < 4; ++i)
        *reinterpret_cast<float4*>(&gt[lrow + i * S::kRW][4 * (lane % LPC)]) =
            make_float4(cur.v[i][0], cur.v[i][1], cur.v[i][2], cur.v[i][3]);
      if (rt == rt0) asm volatile("bar.sync 1, %0;" ::"n"(32 * (kQWarps + 1)) : "memory");
      else asm volatile("bar.sync 3, %0;" ::"n"(32 * kQWarps) : "memory");
      const int nk = nk_s;
      for (int u = threadIdx.x; u < nk * (S::kRows / 4); u += 32 * kQWarps) {
        const int j = u / (S::kRows / 4), g = u % (S::kRows / 4);
        const int col = klist[j];
        const int64_t rq = r0 + 4 * g;
        const float z = kz[j], inv = kinv[j];
        const bool deg = !(inv > 0.0f);
        const uint64_t e = (uint64_t)(cb + col) * (uint64_t)a.M + (uint64_t)rq;
        uint32_t w[4];
        if ((a.M & 3) == 0) {
          const U32x4 p = philox_block(a.c.seed, kStreamSrPcq, e >> 2);
          w[0] = p.x; w[1] = p.y; w[2] = p.z; w[3] = p.w;
        } else {
#pragma unroll
          for (int i = 0; i < 4; ++i) w[i] = philox_word(a.c.seed, kStreamSrPcq, e + i);
        }
        uint32_t word = 0;
#pragma unroll
        for (int i = 0; i < 4; ++i)
          if (rq + i < a.M) word |= sr_code(gt[4 * g + i][col], z, inv, a.c.B, deg, w[i]) << (8 * i);
        tile[j][g] = word;
      }
      asm volatile("bar.sync 2, %0;" ::"n"(32 * kQWarps) : "memory");
      // kept column j: the codes of rows r0 .. r0 + kRows - 1 as 16-byte stores
      for (int t = threadIdx.x; t < nk * (S::kRows / 16); t += 32 * kQWarps) {
        const int j = t / (S::kRows / 16), h = t % (S::kRows / 16);
        const int64_t rb = r0 + 16 * h;
        if (rb < a.M && rb + 16 <= a.c.ld) {
          uint4 val;
          val.x = tile[j][4 * h + 0];
          val.y = tile[j][4 * h + 1];
          val.z = tile[j][4 * h + 2];
          val.w = tile[j][4 * h + 3];
          *reinterpret_cast<uint4*>(a.c.codes + (int64_t)kslot[j] * a.c.ld + rb) = val;
        }
      }
    }
  };
  if (rt0 < row_tiles) quant_load<VEC, S::kRW>(a, rt0 * S::kRows + lrow, c0, cv[0], cur);
  if (PIPE) {
#pragma unroll 1
    for (int64_t rt = rt0; rt < row_tiles; rt += rstep) {
      do_tile(rt);
      cur = nxt;
    }
  } else if (rt0 < row_tiles) {
    do_tile(rt0);
  }
  // a CTA without row tiles (the host never launches one) still meets warp 8's arrive
  if (a.do_pcq && rt0 >= row_tiles) asm volatile("bar.sync 1, %0;" ::"n"(32 * (kQWarps + 1)) : "memory");
}

}  // namespace fqt1

using namespace fqt1;

static bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

static bool valid_params(const fqt1_agp_params* p) {
  return p && (p->bits == 1 || p->bits == 2 || p->bits == 4 || p->bits == 8) && p->mode >= 0 && p->mode <= 2;
}

static bool valid_qgrad(const fqt1_qgrad* q, int64_t min_ld) {
  return q && q->group_min && q->group_range && q->p_hat && q->slot_of_group && q->kept_idx && q->kept_count &&
         q->scale && q->zero && q->codes && q->ld_codes >= min_ld && q->ld_codes % 16 == 0 && aligned16(q->codes);
}

extern "C" size_t fqt1_workspace_size(int32_t which, int64_t M, int64_t D, int64_t K, int32_t rows_per_group) {
  if (which == 0) {
    const int64_t ns = rows_per_group > 0 ? M / rows_per_group : M;
    return (size_t)(2 * ns + 2 * D) * sizeof(uint32_t);
  }
  (void)K;
  return 0;
}

// Resident CTAs on the whole GPU (SMs x CTAs per SM) of a kernel variant, per device; `slot`
// names the variant in the cache (0-3 range pass, 4-7 pipelined quantize pass, 8-11 quantize
// pass one tile per CTA).
template <class Args>
static int resident_wave(void (*k)(Args), int threads, int slot) {
  static std::atomic<int> cache[64][12];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) dev = 0;
  int w = cache[dev][slot].load(std::memory_order_relaxed);
  if (w > 0) return w;
  int sms = 152, per_sm = 1;
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k, threads, 0) != cudaSuccess || per_sm < 1) per_sm = 1;
  w = sms * per_sm;
  cache[dev][slot].store(w, std::memory_order_relaxed);
  return w;
}

// Rows of a contiguous run per CTA so that the CTAs of `cols` column tiles fill about one
// resident wave; the grid's row extent then leaves no CTA without a tile.
static void row_runs(int64_t tiles, int64_t cols, int wave, int64_t* per_cta, int64_t* ctas) {
  const int64_t want = std::max<int64_t>(1, wave / std::max<int64_t>(1, cols));
  *per_cta = (tiles + want - 1) / want;
  if (*per_cta < 1) *per_cta = 1;
  *ctas = std::max<int64_t>(1, (tiles + *per_cta - 1) / *per_cta);
}

// Shared driver of both entry points.
static fqt1_status quantize_impl(const float* g, int64_t M, int64_t D, const float* gamma,
                                 const fqt1_agp_params* ps, fqt1_qgrad* psq, const fqt1_agp_params* pc,
                                 fqt1_qgrad* pcq, void* ws, size_t ws_bytes, int32_t* dev_status, cudaStream_t s) {
  if (!g || M < 1 || D < 1 || !dev_status) return FQT1_ERR_INVALID_ARG;
  if (!aligned16(g) || (gamma && !aligned16(gamma))) return FQT1_ERR_MISALIGNED;
  int64_t rpg = 1, ns = 0;
  if (psq) {
    if (!valid_params(ps) || ps->rows_per_group < 1 || M % ps->rows_per_group != 0) return FQT1_ERR_INVALID_ARG;
    if (!valid_qgrad(psq, fqt1_codes_ld(D))) return FQT1_ERR_INVALID_ARG;
    rpg = ps->rows_per_group;
    ns = M / rpg;
    if (ns > kMaxGroups) return FQT1_ERR_UNSUPPORTED;
  }
  if (pcq) {
    if (!valid_params(pc) || !valid_qgrad(pcq, fqt1_codes_ld(M))) return FQT1_ERR_INVALID_ARG;
    if (D > kMaxGroups) return FQT1_ERR_UNSUPPORTED;
  }
  const size_t need = (size_t)(2 * ns + 2 * D) * sizeof(uint32_t);  // ns = 0 for a channel-only call
  if (!ws || ws_bytes < need) return FQT1_ERR_WORKSPACE;
  if (!aligned16(ws)) return FQT1_ERR_MISALIGNED;
  if (M * D >= (1ll << 46)) return FQT1_ERR_UNSUPPORTED;
  if (M >= (1ll << 31)) return FQT1_ERR_UNSUPPORTED;  // rows go through 32-bit multiply-high division

  uint32_t* smin = static_cast<uint32_t*>(ws);
  uint32_t* cmin = smin + ns;
  uint32_t* smax = cmin + D;
  uint32_t* cmax = smax + ns;
  // min keys and complemented max keys start at 0xFFFFFFFF (fqt1_scq_workspace_init, then the
  // selection kernel of every call resets the keys it read) and both take atomicMin

  const bool vec = (D % 4) == 0;
  RangeArgs ra{g, gamma, M, D, rpg, psq ? smin : nullptr, psq ? smax : nullptr, pcq ? cmin : nullptr,
               pcq ? cmax : nullptr, dev_status, FastDiv((uint32_t)rpg)};
  // lane layout: rows of 8 or 16 lanes when D is that narrow and no warp chunk straddles two
  // sample groups; one resident wave of CTAs at most, each looping over its run of row tiles
  int lpr = 32;
  if (vec && D <= 32 && (!psq || rpg % RangeShape<8>::kChunk == 0)) lpr = 8;
  else if (vec && D <= 64 && (!psq || rpg % RangeShape<16>::kChunk == 0)) lpr = 16;
  void (*rk)(RangeArgs) = lpr == 8 ? range_kernel<8, true>
                        : lpr == 16 ? range_kernel<16, true>
                        : vec ? range_kernel<32, true> : range_kernel<32, false>;
  const int tile = lpr == 8 ? RangeShape<8>::kTile : lpr == 16 ? RangeShape<16>::kTile : RangeShape<32>::kTile;
  const int64_t rcols = (D + 4 * lpr - 1) / (4 * lpr), rtiles = (M + tile - 1) / tile;
  const int wave = resident_wave(rk, 256, lpr == 8 ? 0 : lpr == 16 ? 1 : vec ? 2 : 3);
  int64_t rper = 0, rctas = 0;
  row_runs(rtiles, rcols, wave, &rper, &rctas);
  dim3 rgrid((unsigned)rcols, (unsigned)rctas);
  launch_k(rk, rgrid, dim3(256), 0, s, ra);
  fqt1_count_launches(1);
  FQT1_CUDA_TRY(cudaGetLastError());

  SelectArgs sa[2];
  int nsel = 0;
  int npad_max = 1;
  auto add_sel = [&](const fqt1_agp_params* p, fqt1_qgrad* q, uint32_t* kmin, uint32_t* kmax, int n,
                     uint32_t stream) {
    SelectArgs x;
    x.kmin = kmin; x.kmax = kmax; x.n = n; x.bits = p->bits; x.mode = p->mode;
    x.capacity = (int32_t)fqt1_kept_capacity(n, p->bits, p->mode);
    x.seed = p->seed; x.stream = stream; x.out = *q;
    sa[nsel++] = x;
    int np = 1;
    while (np < n) np <<= 1;
    npad_max = np > npad_max ? np : npad_max;
  };
  if (psq) add_sel(ps, psq, smin, smax, (int)ns, kStreamSelSample);
  if (pcq) add_sel(pc, pcq, cmin, cmax, (int)D, kStreamSelChannel);
  const size_t smem = (size_t)npad_max * 8 + (size_t)npad_max * 4;
  static std::atomic<uint64_t> attr_small{0}, attr_large{0};
  FQT1_CUDA_TRY(smem_attr_once((const void*)select_kernel<256>, kMaxGroups * 12, attr_small));
  FQT1_CUDA_TRY(smem_attr_once((const void*)select_kernel<kSelThreads>, kMaxGroups * 12, attr_large));
  if (npad_max <= 256)  // fewer warps per barrier when every grouping has at most 256 groups
    launch_k(select_kernel<256>, dim3(nsel), dim3(256), smem, s, sa[0], nsel > 1 ? sa[1] : sa[0]);
  else
    launch_k(select_kernel<kSelThreads>, dim3(nsel), dim3(kSelThreads), smem, s, sa[0], nsel > 1 ? sa[1] : sa[0]);
  fqt1_count_launches(1);
  FQT1_CUDA_TRY(cudaGetLastError());

  QuantArgs qa;
  qa.g = g; qa.gamma = gamma; qa.M = M; qa.D = D; qa.rpg = rpg; qa.div_rpg = FastDiv((uint32_t)rpg);
  qa.do_psq = psq != nullptr;
  qa.do_pcq = pcq != nullptr;
  if (psq) qa.s = QBranch{psq->group_min, psq->group_range, psq->slot_of_group, psq->codes, psq->ld_codes,
                          (float)((1 << ps->bits) - 1), ps->seed, psq->kept_idx, psq->kept_count, psq->p_hat,
                          psq->scale, psq->zero};
  else qa.s = QBranch{};
  if (pcq) qa.c = QBranch{pcq->group_min, pcq->group_range, pcq->slot_of_group, pcq->codes, pcq->ld_codes,
                          (float)((1 << pc->bits) - 1), pc->seed, pcq->kept_idx, pcq->kept_count, pcq->p_hat,
                          pcq->scale, pcq->zero};
  else qa.c = QBranch{};
  // tile shape: 16 or 8 lanes per row when D is that narrow.  Tiles that fit in one wave of
  // four CTAs per SM go one per CTA; more tiles go to about one resident wave of pipelined CTAs,
  // each over every gridDim.y-th row tile
  const int lpc = !vec ? 32 : D <= 32 ? 8 : D <= 64 ? 16 : 32;
  const int qrows = lpc == 8 ? QShape<8>::kRows : lpc == 16 ? QShape<16>::kRows : QShape<32>::kRows;
  const int64_t qcols = (D + 4 * lpc - 1) / (4 * lpc), qtiles = (M + qrows - 1) / qrows;
  void (*qk1)(QuantArgs) = lpc == 8 ? quantize_kernel<8, true, false>
                         : lpc == 16 ? quantize_kernel<16, true, false>
                         : vec ? quantize_kernel<32, true, false> : quantize_kernel<32, false, false>;
  void (*qkp)(QuantArgs) = lpc == 8 ? quantize_kernel<8, true, true>
                         : lpc == 16 ? quantize_kernel<16, true, true>
                         : vec ? quantize_kernel<32, true, true> : quantize_kernel<32, false, true>;
  const int vslot = lpc == 8 ? 0 : lpc == 16 ? 1 : vec ? 2 : 3;
  const int wave1 = resident_wave(qk1, 32 * (kQWarps + 1), 8 + vslot);
  const bool pipe = qtiles * qcols > wave1;
  void (*qk)(QuantArgs) = pipe ? qkp : qk1;
  const int qwave = pipe ? resident_wave(qkp, 32 * (kQWarps + 1), 4 + vslot) : wave1;
  const int64_t qctas = std::min<int64_t>(qtiles, std::max<int64_t>(1, qwave / qcols));
  launch_k(qk, dim3((unsigned)qcols, (unsigned)qctas), dim3(32 * (kQWarps + 1)), 0, s, qa);
  fqt1_count_launches(1);
  FQT1_CUDA_TRY(cudaGetLastError());
  return FQT1_OK;
}

extern "C" fqt1_status fqt1_scq_workspace_init(void* ws, size_t ws_bytes, void* stream) {
  if (!ws || ws_bytes == 0) return FQT1_ERR_INVALID_ARG;
  FQT1_CUDA_TRY(cudaMemsetAsync(ws, 0xFF, ws_bytes, (cudaStream_t)stream));
  return FQT1_OK;
}

extern "C" fqt1_status fqt1_agp_quantize_grad(const float* g, int64_t M, int64_t D, int32_t group_axis,
                                              const float* gamma, const fqt1_agp_params* p, fqt1_qgrad* out,
                                              void* ws, size_t ws_bytes, int32_t* dev_status, void* stream) {
  if (group_axis == 0) return quantize_impl(g, M, D, gamma, p, out, nullptr, nullptr, ws, ws_bytes, dev_status,
                                            (cudaStream_t)stream);
  if (group_axis == 1) return quantize_impl(g, M, D, gamma, nullptr, nullptr, p, out, ws, ws_bytes, dev_status,
                                            (cudaStream_t)stream);
  return FQT1_ERR_INVALID_ARG;
}

extern "C" fqt1_status fqt1_scq_quantize(const float* g, int64_t M, int64_t D, const float* gamma,
                                         const fqt1_agp_params* p_sample, const fqt1_agp_params* p_channel,
                                         fqt1_qgrad* psq, fqt1_qgrad* pcq, void* ws, size_t ws_bytes,
                                         int32_t* dev_status, void* stream) {
  if (!psq || !pcq) return FQT1_ERR_INVALID_ARG;
  return quantize_impl(g, M, D, gamma, p_sample, psq, p_channel, pcq, ws, ws_bytes, dev_status,
                       (cudaStream_t)stream);
}

// ---------------------------------------------------------------------------
// Allocation-free variant of fqt1_scq_quantize.
//
// Some callers cannot hand this library a workspace: a plugin interface that
// passes only the input and output tensors, or a training loop whose device
// memory pool is frozen after warm-up so that nothing may call cudaMalloc on
// the step path.  For them the scratch of the range pass (the ordered min / max
// keys of every sample group and channel) lives in a fixed array compiled into
// this library instead of a caller buffer.  The array is shared by every call on
// a device; the first call on the device fills it with 0xFF and every call that
// succeeds leaves it so, like a workspace after fqt1_scq_workspace_init.  A call
// that fails may leave keys behind, so it marks the array for a refill by the next
// call.  Only calls that overlap on the GPU (e.g. on two streams at once)
// interfere, and such calls race.
static __device__ __align__(256) uint32_t g_scq_scratch[FQT1_NOALLOC_SCRATCH_KEYS];

static std::mutex g_scq_scratch_mu;
static void* g_scq_scratch_dev[64];  // device address of g_scq_scratch, per device ordinal
static bool g_scq_scratch_ready[64];  // filled with 0xFF outside a graph capture

// Device address of the scratch array on the calling thread's current device, filled with
// 0xFF on stream s until a fill has run outside a graph capture.  The first call on a device
// looks the address up (cudaGetSymbolAddress) and caches it.  *dev_out is the device ordinal.
static fqt1_status scq_scratch_address(void** out, int* dev_out, cudaStream_t s) {
  int dev = -1;
  FQT1_CUDA_TRY(cudaGetDevice(&dev));
  *dev_out = dev;
  if (dev < 0 || dev >= 64) return FQT1_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_scq_scratch_mu);
  if (!g_scq_scratch_dev[dev]) {
    void* p = nullptr;
    FQT1_CUDA_TRY(cudaGetSymbolAddress(&p, g_scq_scratch));
    g_scq_scratch_dev[dev] = p;
  }
  if (!g_scq_scratch_ready[dev]) {
    cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
    FQT1_CUDA_TRY(cudaStreamIsCapturing(s, &cap));
    FQT1_CUDA_TRY(cudaMemsetAsync(g_scq_scratch_dev[dev], 0xFF, sizeof(g_scq_scratch), s));
    if (cap == cudaStreamCaptureStatusNone) g_scq_scratch_ready[dev] = true;
  }
  *out = g_scq_scratch_dev[dev];
  return FQT1_OK;
}

extern "C" fqt1_status fqt1_scq_quantize_noalloc(const float* g, int64_t M, int64_t D, const float* gamma,
                                                 const fqt1_agp_params* p_sample, const fqt1_agp_params* p_channel,
                                                 fqt1_qgrad* psq, fqt1_qgrad* pcq, int32_t* dev_status,
                                                 void* stream) {
  if (!psq || !pcq || !p_sample || !p_channel || M < 1 || D < 1 || p_sample->rows_per_group < 1)
    return FQT1_ERR_INVALID_ARG;
  const int64_t keys = 2 * (M / p_sample->rows_per_group) + 2 * D;
  if (keys > FQT1_NOALLOC_SCRATCH_KEYS) {
    char msg[200];
    snprintf(msg, sizeof(msg),
             "fqt1_scq_quantize_noalloc: 2*(M/rows_per_group) + 2*D = %lld keys exceed the built-in scratch of %d",
             (long long)keys, (int)FQT1_NOALLOC_SCRATCH_KEYS);
    fqt1_set_error_text(msg);
    return FQT1_ERR_UNSUPPORTED;
  }
  void* scratch = nullptr;
  int dev = -1;
  const fqt1_status st = scq_scratch_address(&scratch, &dev, (cudaStream_t)stream);
  if (st != FQT1_OK) return st;
  const fqt1_status q = quantize_impl(g, M, D, gamma, p_sample, psq, p_channel, pcq, scratch,
                                      sizeof(uint32_t) * FQT1_NOALLOC_SCRATCH_KEYS, dev_status,
                                      (cudaStream_t)stream);
  if (q != FQT1_OK) {
    // the range kernel may have run and left keys that no selection kernel reset: the next
    // call on this device fills the array again
    std::lock_guard<std::mutex> lock(g_scq_scratch_mu);
    g_scq_scratch_ready[dev] = false;
  }
  return q;
}
