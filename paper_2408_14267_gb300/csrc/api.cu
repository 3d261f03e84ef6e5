// C-ABI entry points of the GEMM side, dequantization and the Folder, plus helpers.
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <algorithm>
#include <atomic>

#include "gemm.cuh"

static thread_local char g_last_error[256] = "no error";

void fqt1_set_cuda_error(cudaError_t e) {
  snprintf(g_last_error, sizeof(g_last_error), "%s: %s", cudaGetErrorName(e), cudaGetErrorString(e));
}

extern "C" const char* fqt1_last_cuda_error(void) { return g_last_error; }

void fqt1_set_error_text(const char* msg) { snprintf(g_last_error, sizeof(g_last_error), "%s", msg); }

static std::atomic<int64_t> g_launches{0};
void fqt1_count_launches(int n) { g_launches.fetch_add(n, std::memory_order_relaxed); }
extern "C" int64_t fqt1_kernel_launches(void) { return g_launches.load(std::memory_order_relaxed); }

extern "C" int64_t fqt1_packed_words(int64_t n) { return n < 1 ? 0 : (((n + 31) / 32 + 3) / 4) * 4; }

extern "C" int64_t fqt1_kept_capacity(int64_t n, int32_t bits, int32_t mode) {
  if (n < 1 || bits < 1) return 0;
  if (bits == 1 || mode == FQT1_SEL_BERNOULLI) return n;
  return (n + bits - 1) / bits;
}

extern "C" int64_t fqt1_codes_ld(int64_t n) { return n < 1 ? 0 : ((n + 15) / 16) * 16; }

namespace fqt1 {

// Rows of pruned groups of an [M][K] fp32 output are exactly zero.  Grid: x covers a row in
// chunks of kZeroChunk floats (each thread kZeroVec float4 stores, strided by the block so
// that every store instruction is coalesced), y (and z for more than 65535 rows) the rows.
constexpr int kZeroVec = 8;
constexpr int kZeroChunk = 256 * 4 * kZeroVec;
__global__ void __launch_bounds__(256) zero_pruned_rows_kernel(const int32_t* __restrict__ slot_of_group, int64_t M,
                                                               int64_t K, int64_t rpg, float* __restrict__ out) {
  FQT1_PDL_WAIT();
  FQT1_PDL_TRIGGER();
  const int64_t row = (int64_t)blockIdx.z * 65535 + blockIdx.y;
  if (row >= M || __ldg(slot_of_group + row / rpg) >= 0) return;
  float* dst = out + row * K;
  const int64_t c0 = (int64_t)blockIdx.x * kZeroChunk + threadIdx.x * 4;
  if ((K % 4) == 0) {
#pragma unroll
    for (int v = 0; v < kZeroVec; ++v) {
      const int64_t c = c0 + v * 1024;
      if (c < K) *reinterpret_cast<float4*>(dst + c) = make_float4(0.f, 0.f, 0.f, 0.f);
    }
  } else {
    for (int v = 0; v < kZeroVec; ++v)
      for (int64_t j = c0 + v * 1024; j < c0 + v * 1024 + 4 && j < K; ++j) dst[j] = 0.0f;
  }
}

static void launch_zero_pruned_rows(const int32_t* slot_of_group, int64_t M, int64_t K, int64_t rpg, float* out,
                                    cudaStream_t s) {
  const dim3 grid((unsigned)((K + kZeroChunk - 1) / kZeroChunk), (unsigned)(M < 65535 ? M : 65535),
                  (unsigned)((M + 65534) / 65535));
  launch_k(zero_pruned_rows_kernel, dim3(grid), dim3(256), 0, s, slot_of_group, M, K, rpg, out);
  fqt1_count_launches(1);
}

// out[m, k] = S'_slot * acc[row(m), k] + Z'_slot * cs[k] for rows m of kept groups, 0 otherwise
// (fp32 multiply, multiply, add; no contraction).  Used for dx (groups of rpg rows) and dw (rpg = 1).
__global__ void dequant_rows_kernel(const int32_t* __restrict__ acc, int64_t ldacc,
                                    const int32_t* __restrict__ slot_of_group, const float* __restrict__ scale,
                                    const float* __restrict__ zero, const int32_t* __restrict__ cs, int64_t M,
                                    int64_t K, int64_t rpg, float* __restrict__ out) {
  FQT1_PDL_WAIT();
  FQT1_PDL_TRIGGER();
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= M * K) return;
  const int64_t m = idx / K, k = idx - (idx / K) * K;
  const int64_t g = m / rpg;
  const int32_t sl = __ldg(slot_of_group + g);
  float v = 0.0f;
  if (sl >= 0) {
    const int32_t a = __ldg(acc + ((int64_t)sl * rpg + (m - g * rpg)) * ldacc + k);
    v = __fadd_rn(__fmul_rn(__ldg(scale + sl), __int2float_rn(a)), __fmul_rn(__ldg(zero + sl), __int2float_rn(__ldg(cs + k))));
  }
  out[idx] = v;
}

// Folder of App. C on int32 accumulators + dequantization per sample.
__global__ void col2im_kernel(const int32_t* __restrict__ acc, const int32_t* __restrict__ slot_of_group,
                              const float* __restrict__ scale, const float* __restrict__ zero,
                              const int32_t* __restrict__ cs, int N, int C, int H, int W, int kh, int kw, int stride,
                              int pad, int Ho, int Wo, float* __restrict__ dx) {
  FQT1_PDL_WAIT();
  FQT1_PDL_TRIGGER();
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t total = (int64_t)N * C * H * W;
  if (idx >= total) return;
  const int w = (int)(idx % W);
  const int h = (int)((idx / W) % H);
  const int c = (int)((idx / ((int64_t)W * H)) % C);
  const int n = (int)(idx / ((int64_t)W * H * C));
  const int32_t sl = __ldg(slot_of_group + n);
  float v = 0.0f;
  if (sl >= 0) {
    const int64_t K = (int64_t)C * kh * kw;
    const int64_t rbase = (int64_t)sl * Ho * Wo;
    int32_t a = 0, s = 0;
    for (int i = 0; i < kh; ++i) {
      const int hn = h + pad - i;
      if (hn < 0 || hn % stride) continue;
      const int oh = hn / stride;
      if (oh >= Ho) continue;
      for (int j = 0; j < kw; ++j) {
        const int wn = w + pad - j;
        if (wn < 0 || wn % stride) continue;
        const int ow = wn / stride;
        if (ow >= Wo) continue;
        const int64_t k = ((int64_t)c * kh + i) * kw + j;
        a += __ldg(acc + (rbase + (int64_t)oh * Wo + ow) * K + k);
        s += __ldg(cs + k);
      }
    }
    v = __fadd_rn(__fmul_rn(__ldg(scale + sl), __int2float_rn(a)), __fmul_rn(__ldg(zero + sl), __int2float_rn(s)));
  }
  dx[idx] = v;
}

// Folder with the accumulators staged in shared memory (two kernels).  A CTA owns one kept
// sample, a block of channels and a block of input pixels: it loads, coalesced, the int32
// accumulators of every output pixel whose window touches that block (the k-range of the
// block's channels), then sums the taps of each input pixel from shared memory.  The tile's
// row stride is odd so that neighbouring pixels fall in different banks.
struct FoldArgs {
  const int32_t* acc;
  const int32_t* kept_idx;
  const int32_t* kept_count;
  const float* scale;
  const float* zero;
  const int32_t* cs;
  float* dx;
  int N, C, H, W, kh, kw, stride, pad, Ho, Wo;
  int cb, hb, wb, ncb, nwb, max_rows, max_cols, kstride;
  int64_t K;
  int nhwc;  // dx in memory order N, H, W, C (outputs walked channels fastest) instead of NCHW
};

constexpr int kFoldLoads = 8;  // accumulator loads in flight per thread while staging

// Compact tap lists of a Folder block, so that an input pixel visits only the taps that land on
// it (about (kh / stride) x (kw / stride) of them) instead of testing all kh x kw.  Local row hl
// (input row h0 + hl): taps i whose output row oh = (h0 + hl + pad - i) / stride exists and lies
// in [oh_lo, oh_hi], stored as h_off = (oh - oh_lo) row_pix kstride + i kw (tile offset) and
// h_cs = i kw (column-sum offset), hcnt of them; local column wl likewise: w_off = (ow - ow_lo)
// kstride + j, w_cs = j.  Row wl of the lists holds kh (kw) slots.
__device__ __forceinline__ void fold_tap_lists(const FoldArgs& a, int h0, int nh, int oh_lo, int oh_hi, int row_pix,
                                               int w0, int nw, int ow_lo, int ow_hi, int32_t* h_off, int32_t* h_cs,
                                               int32_t* hcnt, int32_t* w_off, int32_t* w_cs, int32_t* wcnt) {
  for (int hl = threadIdx.x; hl < nh; hl += blockDim.x) {
    int cnt = 0;
    for (int i = 0; i < a.kh; ++i) {
      const int hn = h0 + hl + a.pad - i;
      if (hn < 0 || hn % a.stride) continue;
      const int oh = hn / a.stride;
      if (oh < oh_lo || oh > oh_hi) continue;
      h_off[hl * a.kh + cnt] = (oh - oh_lo) * row_pix * a.kstride + i * a.kw;
      h_cs[hl * a.kh + cnt] = i * a.kw;
      ++cnt;
    }
    hcnt[hl] = cnt;
  }
  for (int wl = threadIdx.x; wl < nw; wl += blockDim.x) {
    int cnt = 0;
    for (int j = 0; j < a.kw; ++j) {
      const int wn = w0 + wl + a.pad - j;
      if (wn < 0 || wn % a.stride) continue;
      const int ow = wn / a.stride;
      if (ow < ow_lo || ow > ow_hi) continue;
      w_off[wl * a.kw + cnt] = (ow - ow_lo) * a.kstride + j;
      w_cs[wl * a.kw + cnt] = j;
      ++cnt;
    }
    wcnt[wl] = cnt;
  }
}

// The integer sum and the folded column sum of one input pixel (local row hl, column wl) of
// channel block offset kc, over its compact tap lists.
__device__ __forceinline__ void fold_pixel(const int32_t* tile, const int32_t* css, const int32_t* h_off,
                                           const int32_t* h_cs, const int32_t* hcnt, const int32_t* w_off,
                                           const int32_t* w_cs, const int32_t* wcnt, int kh, int kw, int hl, int wl,
                                           int kc, int32_t& acc, int32_t& csum) {
  const int hc = hcnt[hl], wc = wcnt[wl];
  const int32_t* ho = h_off + hl * kh;
  const int32_t* hs = h_cs + hl * kh;
  const int32_t* wo = w_off + wl * kw;
  const int32_t* ws = w_cs + wl * kw;
  acc = 0;
  csum = 0;
  for (int p = 0; p < hc; ++p) {
    const int32_t* trow = tile + kc + ho[p];
    const int32_t* crow = css + kc + hs[p];
    for (int q = 0; q < wc; ++q) {
      acc += trow[wo[q]];
      csum += crow[ws[q]];
    }
  }
}

// Folder of a pointwise convolution (1 x 1 window, no padding, stride s): input pixel (h, w)
// receives the tap of output pixel (h / s, w / s) when s divides both, and nothing otherwise.
// A CTA owns one kept sample, one output row oh and 32 channels: it stages the accumulator rows
// of that output row ([Wo][32] ints, coalesced) in shared memory and writes the s input rows
// s oh .. s oh + s - 1 of its channels completely (zeros where no tap lands).
__global__ void __launch_bounds__(256) col2im_pointwise_kernel(FoldArgs a) {
  FQT1_PDL_WAIT();
  FQT1_PDL_TRIGGER();
  extern __shared__ int32_t pw_tile[];  // [32][Wo + 1]
  const int32_t slot = (int32_t)blockIdx.y;
  if (slot >= __ldg(a.kept_count)) return;
  const int n = __ldg(a.kept_idx + slot);
  const int ncb = (a.C + 31) / 32;
  const int oh = blockIdx.x / ncb, c0 = (blockIdx.x - oh * ncb) * 32;
  const int nc = min(32, a.C - c0);
  const int ts = a.Wo + 1;
  const int32_t* src = a.acc + ((int64_t)slot * a.Ho * a.Wo + (int64_t)oh * a.Wo) * a.K + c0;
  for (int e = threadIdx.x; e < a.Wo * 32; e += blockDim.x) {
    const int ow = e >> 5, cl = e & 31;
    pw_tile[cl * ts + ow] = cl < nc ? __ldg(src + (int64_t)ow * a.K + cl) : 0;
  }
  __syncthreads();
  const float sc = __ldg(a.scale + slot), ze = __ldg(a.zero + slot);
  const int h0 = oh * a.stride, h1 = min(a.H, h0 + a.stride);
  const int per = (h1 - h0) * a.W;  // floats of one channel in this CTA's rows
  for (int e = threadIdx.x; e < nc * per; e += blockDim.x) {
    int cl, pos;
    if (a.nhwc) { pos = e / nc; cl = e - pos * nc; }
    else { cl = e / per; pos = e - cl * per; }
    const int hl = pos / a.W, w = pos - hl * a.W;
    float v = 0.0f;
    if (hl == 0 && w % a.stride == 0) {
      const int ow = w / a.stride;
      if (ow < a.Wo)
        v = __fadd_rn(__fmul_rn(sc, __int2float_rn(pw_tile[cl * ts + ow])),
                      __fmul_rn(ze, __int2float_rn(__ldg(a.cs + c0 + cl))));
    }
    if (a.nhwc)
      a.dx[(((int64_t)n * a.H + h0 + hl) * a.W + w) * a.C + c0 + cl] = v;
    else
      a.dx[(((int64_t)n * a.C + c0 + cl) * a.H + h0 + hl) * a.W + w] = v;
  }
}

// Folder over whole input rows (blocks of at least min(C, 4) channels): a CTA owns channels
// [c0, c0+cb) and input rows [h0, h0+hb) of its sample; each warp copies the accumulator
// k-range of one output pixel at a time, which is coalesced when that range is long.
__global__ void __launch_bounds__(256) col2im_rows_kernel(FoldArgs a) {
  FQT1_PDL_WAIT();
  FQT1_PDL_TRIGGER();
  extern __shared__ int32_t fold_smem[];
  const int32_t slot = (int32_t)blockIdx.y;  // one kept sample per grid row
  if (slot >= __ldg(a.kept_count)) return;
  const int n = __ldg(a.kept_idx + slot);
  const int cblk = blockIdx.x % a.ncb, hblk = blockIdx.x / a.ncb;
  const int c0 = cblk * a.cb, h0 = hblk * a.hb;
  const int c1 = min(a.C, c0 + a.cb), h1 = min(a.H, h0 + a.hb);
  const int nc = c1 - c0, nh = h1 - h0;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int plane = nh * a.W;  // contiguous floats of one channel inside the block
  const int khw = a.kh * a.kw;
  int oh_lo = h0 + a.pad - (a.kh - 1);
  oh_lo = oh_lo <= 0 ? 0 : (oh_lo + a.stride - 1) / a.stride;
  const int oh_hi = min(a.Ho - 1, (h1 - 1 + a.pad) / a.stride);
  const int nrows = oh_hi - oh_lo + 1;
  const int kb = nc * khw;
  int32_t* tile = fold_smem;                                   // [max_rows * Wo][kstride]
  int32_t* h_off = tile + a.max_rows * a.Wo * a.kstride;       // [hb][kh] tap lists of the rows
  int32_t* h_cs = h_off + a.hb * a.kh;
  int32_t* hcnt = h_cs + a.hb * a.kh;                          // [hb]
  int32_t* w_off = hcnt + a.hb;                                // [W][kw] tap lists of the columns
  int32_t* w_cs = w_off + a.W * a.kw;
  int32_t* wcnt = w_cs + a.W * a.kw;                           // [W]
  int32_t* css = wcnt + a.W;                                   // [cb * khw]: colsum of the block
  fold_tap_lists(a, h0, nh, oh_lo, oh_hi, a.Wo, 0, a.W, 0, a.Wo - 1, h_off, h_cs, hcnt, w_off, w_cs, wcnt);
  const int64_t kbase = (int64_t)c0 * khw;
  for (int x = threadIdx.x; x < kb; x += blockDim.x) css[x] = __ldg(a.cs + kbase + x);
  if (nrows > 0) {
    // one accumulator row segment (kb ints) per warp iteration; 8 loads in flight per lane
    const int npix = nrows * a.Wo;
    const int64_t rbase = (int64_t)slot * a.Ho * a.Wo + (int64_t)oh_lo * a.Wo;
    for (int pix = warp; pix < npix; pix += blockDim.x >> 5) {
      const int32_t* src = a.acc + (rbase + pix) * a.K + kbase;
      int32_t* dst = tile + pix * a.kstride;
      for (int k0 = 0; k0 < kb; k0 += 256) {
        int32_t v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int kk = k0 + 32 * u + lane;
          v[u] = kk < kb ? __ldg(src + kk) : 0;
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int kk = k0 + 32 * u + lane;
          if (kk < kb) dst[kk] = v[u];
        }
      }
    }
  }
  __syncthreads();
  const float sc = __ldg(a.scale + slot), ze = __ldg(a.zero + slot);
  const FastDiv div_plane((uint32_t)plane), div_w((uint32_t)a.W), div_nc((uint32_t)nc);
  for (int e = threadIdx.x; e < nc * plane; e += blockDim.x) {  // output (channel, row, column) of the block
    int cl, pos;
    if (a.nhwc) {  // channels fastest: a pixel's nc channels are contiguous in dx
      pos = (int)div_nc.div((uint32_t)e);
      cl = e - pos * nc;
    } else {
      cl = (int)div_plane.div((uint32_t)e);
      pos = e - cl * plane;
    }
    const int hl = (int)div_w.div((uint32_t)pos), w = pos - hl * a.W;
    int32_t acc, csum;
    fold_pixel(tile, css, h_off, h_cs, hcnt, w_off, w_cs, wcnt, a.kh, a.kw, hl, w, cl * khw, acc, csum);
    const float v = __fadd_rn(__fmul_rn(sc, __int2float_rn(acc)), __fmul_rn(ze, __int2float_rn(csum)));
    if (a.nhwc)
      a.dx[(((int64_t)n * a.H + h0 + hl) * a.W + w) * a.C + c0 + cl] = v;
    else
      a.dx[(((int64_t)n * a.C + c0 + cl) * a.H + h0 + hl) * a.W + w] = v;
  }
}

// Folder over blocks of input rows and columns (shapes whose whole-row blocks would hold fewer
// than min(C, 4) channels, such as the 7 x 7 stride-2 stem on 3 channels): a CTA owns channels
// [c0, c0+cb), rows [h0, h0+hb) and columns [w0, w0+wb) of its sample, which keeps the staged
// halo of large, strided windows small; the staging loop walks the (pixel, k) elements of the
// halo with every thread's loads in flight together, whatever the length of a pixel's k-range.
__global__ void __launch_bounds__(256) col2im_tiled_kernel(FoldArgs a) {
  FQT1_PDL_WAIT();
  FQT1_PDL_TRIGGER();
  extern __shared__ int32_t fold_smem[];
  const int32_t slot = (int32_t)blockIdx.y;  // one kept sample per grid row
  if (slot >= __ldg(a.kept_count)) return;
  const int n = __ldg(a.kept_idx + slot);
  const int cblk = blockIdx.x % a.ncb, rest = blockIdx.x / a.ncb;
  const int wblk = rest % a.nwb, hblk = rest / a.nwb;
  const int c0 = cblk * a.cb, h0 = hblk * a.hb, w0 = wblk * a.wb;
  const int c1 = min(a.C, c0 + a.cb), h1 = min(a.H, h0 + a.hb), w1 = min(a.W, w0 + a.wb);
  const int nc = c1 - c0, nh = h1 - h0, nw = w1 - w0;
  const int khw = a.kh * a.kw;
  // output rows / columns whose windows reach the block
  int oh_lo = h0 + a.pad - (a.kh - 1);
  oh_lo = oh_lo <= 0 ? 0 : (oh_lo + a.stride - 1) / a.stride;
  const int oh_hi = min(a.Ho - 1, (h1 - 1 + a.pad) / a.stride);
  int ow_lo = w0 + a.pad - (a.kw - 1);
  ow_lo = ow_lo <= 0 ? 0 : (ow_lo + a.stride - 1) / a.stride;
  const int ow_hi = min(a.Wo - 1, (w1 - 1 + a.pad) / a.stride);
  const int nrows = oh_hi - oh_lo + 1, ncols = ow_hi - ow_lo + 1;
  const int kb = nc * khw;
  int32_t* tile = fold_smem;                                   // [max_rows * max_cols][kstride]
  int32_t* h_off = tile + a.max_rows * a.max_cols * a.kstride; // [hb][kh] tap lists of the rows
  int32_t* h_cs = h_off + a.hb * a.kh;
  int32_t* hcnt = h_cs + a.hb * a.kh;                          // [hb]
  int32_t* w_off = hcnt + a.hb;                                // [wb][kw] tap lists of the columns
  int32_t* w_cs = w_off + a.wb * a.kw;
  int32_t* wcnt = w_cs + a.wb * a.kw;                          // [wb]
  int32_t* css = wcnt + a.wb;                                  // [cb * khw]: colsum of the block
  fold_tap_lists(a, h0, nh, oh_lo, oh_hi, a.max_cols, w0, nw, ow_lo, ow_hi, h_off, h_cs, hcnt, w_off, w_cs, wcnt);
  const int64_t kbase = (int64_t)c0 * khw;
  for (int x = threadIdx.x; x < kb; x += blockDim.x) css[x] = __ldg(a.cs + kbase + x);
  if (nrows > 0 && ncols > 0) {
    // the (pixel, k) elements of the halo, kFoldLoads loads in flight per thread whatever kb is
    const int total = nrows * ncols * kb;
    const FastDiv div_kb((uint32_t)kb), div_cols((uint32_t)ncols);
    // the halo's first accumulator of the block: offsets from it fit 32 bits (a halo row of
    // pixels spans at most Wo K words)
    const int32_t* src0 = a.acc + ((int64_t)slot * a.Ho * a.Wo + (int64_t)oh_lo * a.Wo + ow_lo) * a.K + kbase;
    const int rowK = a.Wo * (int)a.K, K32 = (int)a.K;
    if ((kb & 3) == 0 && (K32 & 3) == 0 && (kbase & 3) == 0) {
      // k-ranges of whole 16-byte groups: one 16-byte load per four elements (a quarter of the
      // index arithmetic), stored as four words (the tile's row stride is odd)
      const int kb4 = kb >> 2, total4 = total >> 2;
      const FastDiv div_kb4((uint32_t)kb4);
      for (int e0 = threadIdx.x; e0 < total4; e0 += blockDim.x * kFoldLoads) {
        int4 v[kFoldLoads];
        int dsti[kFoldLoads];
#pragma unroll
        for (int u = 0; u < kFoldLoads; ++u) {
          const int e = min(e0 + u * (int)blockDim.x, total4 - 1);  // clamped: every load is valid
          const int pix = (int)div_kb4.div((uint32_t)e), kk = 4 * (e - pix * kb4);
          const int r = (int)div_cols.div((uint32_t)pix), cl = pix - r * ncols;
          v[u] = __ldg(reinterpret_cast<const int4*>(src0 + r * rowK + cl * K32 + kk));
          dsti[u] = (r * a.max_cols + cl) * a.kstride + kk;
        }
#pragma unroll
        for (int u = 0; u < kFoldLoads; ++u) {
          if (e0 + u * (int)blockDim.x >= total4) break;
          int32_t* d = tile + dsti[u];
          d[0] = v[u].x; d[1] = v[u].y; d[2] = v[u].z; d[3] = v[u].w;
        }
      }
    } else
    for (int e0 = threadIdx.x; e0 < total; e0 += blockDim.x * kFoldLoads) {
      int32_t v[kFoldLoads];
      int dsti[kFoldLoads];
#pragma unroll
      for (int u = 0; u < kFoldLoads; ++u) {
        const int e = min(e0 + u * (int)blockDim.x, total - 1);  // clamped: every load is valid
        const int pix = (int)div_kb.div((uint32_t)e), kk = e - pix * kb;
        const int r = (int)div_cols.div((uint32_t)pix), cl = pix - r * ncols;
        v[u] = __ldg(src0 + r * rowK + cl * K32 + kk);
        dsti[u] = (r * a.max_cols + cl) * a.kstride + kk;
      }
#pragma unroll
      for (int u = 0; u < kFoldLoads; ++u)
        if (e0 + u * (int)blockDim.x < total) tile[dsti[u]] = v[u];
    }
  }
  __syncthreads();
  const float sc = __ldg(a.scale + slot), ze = __ldg(a.zero + slot);
  const int plane = nh * nw;
  const FastDiv div_plane((uint32_t)plane), div_w((uint32_t)nw), div_nc((uint32_t)nc);
  for (int e = threadIdx.x; e < nc * plane; e += blockDim.x) {  // output (channel, row, column) of the block
    int cl, pos;
    if (a.nhwc) {  // channels fastest: a pixel's nc channels are contiguous in dx
      pos = (int)div_nc.div((uint32_t)e);
      cl = e - pos * nc;
    } else {
      cl = (int)div_plane.div((uint32_t)e);
      pos = e - cl * plane;
    }
    const int hl = (int)div_w.div((uint32_t)pos), wl = pos - hl * nw;
    int32_t acc, csum;
    fold_pixel(tile, css, h_off, h_cs, hcnt, w_off, w_cs, wcnt, a.kh, a.kw, hl, wl, cl * khw, acc, csum);
    const float v = __fadd_rn(__fmul_rn(sc, __int2float_rn(acc)), __fmul_rn(ze, __int2float_rn(csum)));
    if (a.nhwc)
      a.dx[(((int64_t)n * a.H + h0 + hl) * a.W + w0 + wl) * a.C + c0 + cl] = v;
    else
      a.dx[(((int64_t)n * a.C + c0 + cl) * a.H + h0 + hl) * a.W + w0 + wl] = v;
  }
}

// Folder on column-major accumulators (the layout fqt1_bwd_input_gemm_colmajor writes; T int32,
// or int16 where every sum fits): acc[k * ld + r] for kept row r = slot Ho Wo + oh Wo + ow and
// column k = c kh kw + i kw + j; the tap sums are taken in int32.
// A thread owns elements e = c H W + h W + w of one kept sample's dx plane; tap (i, j) of input
// pixel (h, w) is the accumulator of output pixel oh = (h + pad - i) / stride,
// ow = (w + pad - j) / stride when both divisions are exact and land in the output map.  The 32
// lanes of a warp hold consecutive elements, so for each tap they read consecutive rows of one
// column: every load is coalesced and nothing is staged.  KH, KW, S: compile-time window and
// stride (0: taken from the arguments).
struct FoldCmArgs {
  const void* acc;  // int32 or int16 (the kernel's T)
  int64_t ld;
  const int32_t* kept_idx;
  const int32_t* kept_count;
  const float* scale;
  const float* zero;
  const int32_t* cs;
  float* dx;
  int H, W, kh, kw, stride, pad, Ho, Wo;
  int64_t plane;  // C H W floats of one sample
  FastDiv div_hw, div_w;
  int K;          // C kh kw columns
  int cs_smem;    // 1: the column sums are staged in shared memory (K <= 12288)
};

// Elements per thread of col2im_colmajor_kernel<KH, KW, S>: 4 for a runtime window, else by the
// number c of tap candidates (a thread holds U c loaded accumulators): 1 for c >= 16, 2 for
// c >= 4, 4 below (64 registers, 4 CTAs per SM).  The launcher sizes its grid with the same
// function.
__host__ __device__ constexpr int fold_cm_cand(int KH, int KW, int S) {
  return ((KH + S - 1) / S) * ((KW + S - 1) / S);
}
__host__ __device__ constexpr int fold_cm_per(int KH, int KW, int S) {
  return KH == 0 ? 4
                 : (fold_cm_cand(KH, KW, S) >= 16 ? 1 : (fold_cm_cand(KH, KW, S) >= 4 ? 2 : 4));
}

template <int KH, int KW, int S, class T>
__global__ void __launch_bounds__(256, 4) col2im_colmajor_kernel(FoldCmArgs a) {
  // With a compile-time window, an input pixel's taps are enumerated by residue: row taps
  // i = rh + S mi (rh = (h + pad) mod S) land on output row oh = qh - mi (qh = (h + pad) / S),
  // columns likewise, so only ceil(KH / S) ceil(KW / S) candidates exist (3 x 3 stride 1: 9,
  // 7 x 7 stride 2: 16).  Every candidate's load is issued unconditionally from a clamped,
  // valid address and masked afterwards, so a thread's loads are all in flight together; the
  // column sums of the taps come from shared memory afterwards.
  constexpr int SS = S > 0 ? S : 1;  // the compile-time stride (1 for a runtime window)
  constexpr int CI = KH ? (KH + SS - 1) / SS : 1, CJ = KW ? (KW + SS - 1) / SS : 1;
  constexpr int U = fold_cm_per(KH, KW, SS);  // elements per thread
  extern __shared__ int32_t fold_cs[];        // [K] column sums when a.cs_smem
  FQT1_PDL_WAIT();
  FQT1_PDL_TRIGGER();
  const int kh = KH ? KH : a.kh, kw = KW ? KW : a.kw, st = S ? S : a.stride;
  const int khw = kh * kw, HW = a.H * a.W;
  const int32_t* csb = a.cs;
  if (a.cs_smem) {
    for (int k = threadIdx.x; k < a.K; k += blockDim.x) fold_cs[k] = __ldg(a.cs + k);
    __syncthreads();
    csb = fold_cs;
  }
  // grid rows loop over the kept slots (the grid is sized by occupancy, not by the samples, so
  // few CTAs are launched only to find their sample pruned)
  const int kept = __ldg(a.kept_count);
  for (int slot = (int)blockIdx.y; slot < kept; slot += (int)gridDim.y) {
    const int n = __ldg(a.kept_idx + slot);
    const T* accs = static_cast<const T*>(a.acc) + (int64_t)slot * a.Ho * a.Wo;
    const float sc = __ldg(a.scale + slot), ze = __ldg(a.zero + slot);
    const int64_t e0 = (int64_t)blockIdx.x * (256 * U) + threadIdx.x;
    int32_t av[U], cv[U];
    if (KH) {
      int32_t va[U][CI * CJ];
      uint32_t ok[U];
      int cbase[U], rhv[U], rwv[U];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int64_t e = min(e0 + u * 256, a.plane - 1);  // clamped: every address is valid
        const int c = (int)a.div_hw.div((uint32_t)e), pix = (int)e - c * HW;
        const int h = (int)a.div_w.div((uint32_t)pix), w = pix - h * a.W;
        const T* col = accs + (int64_t)c * khw * a.ld;
        const int hp = h + a.pad, wp = w + a.pad;
        const int rh = SS == 1 ? 0 : hp % SS, qh = SS == 1 ? hp : hp / SS;
        const int rw = SS == 1 ? 0 : wp % SS, qw = SS == 1 ? wp : wp / SS;
        cbase[u] = c * khw;
        rhv[u] = rh;
        rwv[u] = rw;
        uint32_t m = 0;
#pragma unroll
        for (int mi = 0; mi < CI; ++mi) {
          const int i = rh + SS * mi, oh = qh - mi;
          const bool vi = i < KH && oh >= 0 && oh < a.Ho;
#pragma unroll
          for (int mj = 0; mj < CJ; ++mj) {
            const int j = rw + SS * mj, ow = qw - mj;
            const bool v = vi && j < KW && ow >= 0 && ow < a.Wo;
            m |= v ? 1u << (mi * CJ + mj) : 0u;
            va[u][mi * CJ + mj] = (int32_t)__ldg(col + (v ? (int64_t)(i * KW + j) * a.ld + oh * a.Wo + ow : 0));
          }
        }
        ok[u] = m;
      }
#pragma unroll
      for (int u = 0; u < U; ++u) {
        int32_t sa = 0, sc_ = 0;
#pragma unroll
        for (int mi = 0; mi < CI; ++mi) {
#pragma unroll
          for (int mj = 0; mj < CJ; ++mj) {
            const bool v = (ok[u] >> (mi * CJ + mj)) & 1u;
            const int t = (rhv[u] + SS * mi) * KW + rwv[u] + SS * mj;
            sa += v ? va[u][mi * CJ + mj] : 0;
            sc_ += v ? csb[cbase[u] + t] : 0;
          }
        }
        av[u] = sa;
        cv[u] = sc_;
      }
    } else {
      // runtime window: every tap tested in turn
#pragma unroll
      for (int u = 0; u < U; ++u) {
        av[u] = 0;
        cv[u] = 0;
        const int64_t e = e0 + u * 256;
        if (e >= a.plane) continue;
        const int c = (int)a.div_hw.div((uint32_t)e), pix = (int)e - c * HW;
        const int h = (int)a.div_w.div((uint32_t)pix), w = pix - h * a.W;
        const T* col = accs + (int64_t)c * khw * a.ld;
        const int32_t* csc = csb + c * khw;
#pragma unroll 1
        for (int i = 0; i < kh; ++i) {
          const int hn = h + a.pad - i;
          if (hn < 0) break;  // decreasing in i
          if (hn % st) continue;
          const int oh = hn / st;
          if (oh >= a.Ho) continue;
#pragma unroll 1
          for (int j = 0; j < kw; ++j) {
            const int wn = w + a.pad - j;
            if (wn < 0) break;
            if (wn % st) continue;
            const int ow = wn / st;
            if (ow >= a.Wo) continue;
            const int t = i * kw + j;
            av[u] += (int32_t)__ldg(col + (int64_t)t * a.ld + oh * a.Wo + ow);
            cv[u] += csc[t];
          }
        }
      }
    }
    float* out = a.dx + (int64_t)n * a.plane;
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int64_t e = e0 + u * 256;
      if (e < a.plane)
        out[e] = __fadd_rn(__fmul_rn(sc, __int2float_rn(av[u])), __fmul_rn(ze, __int2float_rn(cv[u])));
    }
  }  // kept slots
}

// The same Folder with dx channels-last (dx[n, h, w, c]): a CTA owns 32 consecutive positions
// p = h W + w of a kept sample's plane and 32 channels.  Lane l of warp w holds position l and
// channels 4 w .. 4 w + 3, so each position's tap candidates and their validity are worked out
// once, and each tap's loads run along the 32 positions of a column (coalesced); the 32 x 32
// block of results then turns through shared memory into 128-byte channel runs.
template <int KH, int KW, int S, class T>
__global__ void __launch_bounds__(256, 2) col2im_colmajor_nhwc_kernel(FoldCmArgs a) {
  constexpr int SS = S > 0 ? S : 1;
  constexpr int CI = KH ? (KH + SS - 1) / SS : 1, CJ = KW ? (KW + SS - 1) / SS : 1;
  constexpr int NCAND = CI * CJ;
  constexpr int CPW = 4;   // channels per warp
  constexpr int CB = 2;    // channels whose loads are in flight together
  extern __shared__ int32_t fold_cs[];  // [K] column sums when a.cs_smem
  __shared__ float blk[32][33];         // [channel in block][position in block]
  FQT1_PDL_WAIT();
  FQT1_PDL_TRIGGER();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int kh = KH ? KH : a.kh, kw = KW ? KW : a.kw, st = S ? S : a.stride;
  const int khw = kh * kw, HW = a.H * a.W, C = (int)(a.plane / HW);
  const int32_t* csb = a.cs;
  if (a.cs_smem) {
    for (int k = threadIdx.x; k < a.K; k += blockDim.x) fold_cs[k] = __ldg(a.cs + k);
    __syncthreads();
    csb = fold_cs;
  }
  const int npb = (HW + 31) / 32;
  const int pb = (int)(blockIdx.x % npb), cblk = (int)(blockIdx.x / npb);
  const int pos = min(pb * 32 + lane, HW - 1);  // clamped: every address below is valid
  const int h = (int)a.div_w.div((uint32_t)pos), w = pos - h * a.W;
  // this position's tap candidates (compile-time window: by residue, as the NCHW kernel)
  int toff[NCAND], tix[NCAND];
  uint32_t ok = 0;
  if (KH) {
    const int hp = h + a.pad, wp = w + a.pad;
    const int rh = SS == 1 ? 0 : hp % SS, qh = SS == 1 ? hp : hp / SS;
    const int rw = SS == 1 ? 0 : wp % SS, qw = SS == 1 ? wp : wp / SS;
#pragma unroll
    for (int mi = 0; mi < CI; ++mi) {
      const int i = rh + SS * mi, oh = qh - mi;
      const bool vi = i < KH && oh >= 0 && oh < a.Ho;
#pragma unroll
      for (int mj = 0; mj < CJ; ++mj) {
        const int j = rw + SS * mj, ow = qw - mj;
        const bool v = vi && j < KW && ow >= 0 && ow < a.Wo;
        ok |= v ? 1u << (mi * CJ + mj) : 0u;
        toff[mi * CJ + mj] = v ? oh * a.Wo + ow : 0;
        tix[mi * CJ + mj] = v ? i * KW + j : 0;
      }
    }
  }
  const int c_base = cblk * 32 + warp * CPW;
  const int kept = __ldg(a.kept_count);
  for (int slot = (int)blockIdx.y; slot < kept; slot += (int)gridDim.y) {
    const int n = __ldg(a.kept_idx + slot);
    const T* accs = static_cast<const T*>(a.acc) + (int64_t)slot * a.Ho * a.Wo;
    const float sc = __ldg(a.scale + slot), ze = __ldg(a.zero + slot);
#pragma unroll
    for (int u0 = 0; u0 < CPW; u0 += CB) {
      int32_t av[CB], cv[CB];
      if (KH) {
        int32_t va[CB][NCAND];
#pragma unroll
        for (int u = 0; u < CB; ++u) {
          const int c = min(c_base + u0 + u, C - 1);
          const T* col = accs + (int64_t)c * khw * a.ld;
#pragma unroll
          for (int x = 0; x < NCAND; ++x) va[u][x] = (int32_t)__ldg(col + (int64_t)tix[x] * a.ld + toff[x]);
        }
#pragma unroll
        for (int u = 0; u < CB; ++u) {
          const int c = min(c_base + u0 + u, C - 1);
          int32_t sa = 0, sc_ = 0;
#pragma unroll
          for (int x = 0; x < NCAND; ++x) {
            const bool v = (ok >> x) & 1u;
            sa += v ? va[u][x] : 0;
            sc_ += v ? csb[c * khw + tix[x]] : 0;
          }
          av[u] = sa;
          cv[u] = sc_;
        }
      } else {
        // runtime window: every tap tested in turn
#pragma unroll
        for (int u = 0; u < CB; ++u) {
          av[u] = 0;
          cv[u] = 0;
          const int c = min(c_base + u0 + u, C - 1);
          const T* col = accs + (int64_t)c * khw * a.ld;
#pragma unroll 1
          for (int i = 0; i < kh; ++i) {
            const int hn = h + a.pad - i;
            if (hn < 0) break;
            if (hn % st) continue;
            const int oh = hn / st;
            if (oh >= a.Ho) continue;
#pragma unroll 1
            for (int j = 0; j < kw; ++j) {
              const int wn = w + a.pad - j;
              if (wn < 0) break;
              if (wn % st) continue;
              const int ow = wn / st;
              if (ow >= a.Wo) continue;
              const int t = i * kw + j;
              av[u] += (int32_t)__ldg(col + (int64_t)t * a.ld + oh * a.Wo + ow);
              cv[u] += csb[c * khw + t];
            }
          }
        }
      }
#pragma unroll
      for (int u = 0; u < CB; ++u)
        blk[warp * CPW + u0 + u][lane] =
            __fadd_rn(__fmul_rn(sc, __int2float_rn(av[u])), __fmul_rn(ze, __int2float_rn(cv[u])));
    }
    __syncthreads();
    // positions 4 w .. 4 w + 3 of the block, lane = channel: 128-byte runs of dx[n, p, :]
    float* out = a.dx + (int64_t)n * a.plane;
    const int c = cblk * 32 + lane;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int p = pb * 32 + warp * 4 + q;
      if (p < HW && c < C) out[(int64_t)p * C + c] = blk[lane][warp * 4 + q];
    }
    __syncthreads();
  }
}

}  // namespace fqt1

using namespace fqt1;

static bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

// Output extent of a convolution along one axis, (n + 2 pad - k) / stride + 1 for n, k, stride
// >= 1 and pad >= 0, computed in 64 bits: 0 when the window does not fit, -1 when n + 2 pad
// does not fit an int (the kernels' index arithmetic is 32-bit).
static int64_t conv_extent(int32_t n, int32_t k, int32_t stride, int32_t pad) {
  const int64_t span = (int64_t)n + 2 * (int64_t)pad;
  if (span >= (1ll << 31)) return -1;
  return span < k ? 0 : (span - k) / stride + 1;
}

// SMs of the current device (cached per device ordinal; 152 if the query fails)
static int sm_count_api() {
  static std::atomic<int> cache[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 152;
  int v = cache[dev].load(std::memory_order_relaxed);
  if (v > 0) return v;
  if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v < 1) v = 152;
  cache[dev].store(v, std::memory_order_relaxed);
  return v;
}
static bool valid_bits(int b) { return b == 1 || b == 2 || b == 4 || b == 8; }

extern "C" fqt1_status fqt1_fwd_gemm_bias(const uint32_t* sx_row, const uint32_t* sw_row, int64_t M, int64_t D,
                                          int64_t K, const float* gamma, const float* bias, int32_t* acc, float* y,
                                          void* stream) {
  if (!sx_row || !sw_row || M < 1 || D < 1 || K < 1 || (!acc && !y) || (y && !gamma) || (bias && !y))
    return FQT1_ERR_INVALID_ARG;
  if (!aligned16(sx_row) || !aligned16(sw_row) || (acc && !aligned16(acc)) || (y && !aligned16(y)) ||
      (gamma && !aligned16(gamma)) || (bias && !aligned16(bias)))
    return FQT1_ERR_MISALIGNED;
  if (K >= (1ll << 24) || (M + 63) / 64 > 65535) return FQT1_ERR_UNSUPPORTED;
  FQT1_CUDA_TRY(launch_fwd_tc(sx_row, sw_row, M, D, K, gamma, bias, acc, y, nullptr, (cudaStream_t)stream));
  return FQT1_OK;
}

extern "C" fqt1_status fqt1_fwd_gemm_e4m3w(const uint32_t* sx_row, const uint8_t* w_e4m3, int64_t ld_w, int64_t M,
                                           int64_t D, int64_t K, const float* gamma, const float* bias, int32_t* acc,
                                           float* y, void* stream) {
  if (!sx_row || !w_e4m3 || !gamma || !y || M < 1 || D < 1 || K < 1 || ld_w < K || ld_w % 16)
    return FQT1_ERR_INVALID_ARG;
  if (!aligned16(sx_row) || !aligned16(w_e4m3) || (acc && !aligned16(acc)) || !aligned16(y) || !aligned16(gamma) ||
      (bias && !aligned16(bias)))
    return FQT1_ERR_MISALIGNED;
  if (K >= (1ll << 24) || (M + 63) / 64 > 65535) return FQT1_ERR_UNSUPPORTED;
  FQT1_CUDA_TRY(launch_fwd_e4m3w_tc(sx_row, w_e4m3, ld_w, M, D, K, gamma, bias, acc, y, nullptr, (cudaStream_t)stream));
  return FQT1_OK;
}

extern "C" fqt1_status fqt1_test_expired_wait(const uint32_t* sx_row, const uint32_t* sw_row, int64_t M, int64_t D,
                                              int64_t K, const float* gamma, float* y, int32_t* dev_status,
                                              void* stream) {
  if (!sx_row || !sw_row || !gamma || !y || !dev_status || M < 1 || D < 1 || K < 1) return FQT1_ERR_INVALID_ARG;
  if (!aligned16(sx_row) || !aligned16(sw_row) || !aligned16(gamma) || !aligned16(y)) return FQT1_ERR_MISALIGNED;
  if (K >= (1ll << 24) || (M + 127) / 128 > 65535) return FQT1_ERR_UNSUPPORTED;
  FQT1_CUDA_TRY(launch_fwd_lost_arrive_tc(sx_row, sw_row, M, D, K, gamma, y, dev_status, (cudaStream_t)stream));
  return FQT1_OK;
}

extern "C" fqt1_status fqt1_fwd_gemm(const uint32_t* sx_row, const uint32_t* sw_row, int64_t M, int64_t D,
                                     int64_t K, const float* gamma, int32_t* acc, float* y, void* stream) {
  return fqt1_fwd_gemm_bias(sx_row, sw_row, M, D, K, gamma, nullptr, acc, y, stream);
}

extern "C" int32_t fqt1_conv_implicit_supported(int32_t N, int32_t C, int32_t H, int32_t W, int32_t kh, int32_t kw,
                                                int32_t stride, int32_t pad) {
  return implicit_conv_supported(N, C, H, W, kh, kw, stride, pad) ? 1 : 0;
}

extern "C" fqt1_status fqt1_conv_fwd_implicit(const uint32_t* x_pix, const uint32_t* w_taps, int32_t N, int32_t C,
                                              int32_t H, int32_t W, int32_t kh, int32_t kw, int32_t stride,
                                              int32_t pad, int64_t D, const float* gamma, const float* bias,
                                              int32_t* acc, float* y, void* stream) {
  if (!x_pix || !w_taps || !gamma || !y || N < 1 || C < 1 || H < 1 || W < 1 || kh < 1 || kw < 1 || stride < 1 ||
      pad < 0 || D < 1)
    return FQT1_ERR_INVALID_ARG;
  if (!aligned16(x_pix) || !aligned16(w_taps) || !aligned16(gamma) || !aligned16(y) || (acc && !aligned16(acc)) ||
      (bias && !aligned16(bias)))
    return FQT1_ERR_MISALIGNED;
  if (!implicit_conv_supported(N, C, H, W, kh, kw, stride, pad)) return FQT1_ERR_UNSUPPORTED;
  FQT1_CUDA_TRY(launch_fwd_implicit_tc(x_pix, w_taps, N, C, H, W, kh, pad, D, gamma, bias, acc, y, nullptr,
                                       (cudaStream_t)stream));
  return FQT1_OK;
}

extern "C" fqt1_status fqt1_bwd_input_gemm(const fqt1_qgrad* psq, const uint32_t* sw_col, const int32_t* colsum_w,
                                           int64_t M, int64_t D, int64_t K, const fqt1_agp_params* p,
                                           int32_t* acc, float* dx, void* stream) {
  if (!psq || !sw_col || !p || M < 1 || D < 1 || K < 1 || (!acc && !dx)) return FQT1_ERR_INVALID_ARG;
  if (!valid_bits(p->bits) || p->rows_per_group < 1 || M % p->rows_per_group) return FQT1_ERR_INVALID_ARG;
  if (dx && !colsum_w) return FQT1_ERR_INVALID_ARG;
  if (colsum_w && !aligned16(colsum_w)) return FQT1_ERR_MISALIGNED;
  if (!psq->codes || !psq->kept_count || !psq->slot_of_group || !psq->scale || !psq->zero ||
      psq->ld_codes < fqt1_codes_ld(D) || psq->ld_codes % 16)
    return FQT1_ERR_INVALID_ARG;
  if (!aligned16(sw_col) || (acc && !aligned16(acc)) || (dx && !aligned16(dx))) return FQT1_ERR_MISALIGNED;
  const int64_t rpg = p->rows_per_group;
  const int64_t cap_rows = fqt1_kept_capacity(M / rpg, p->bits, p->mode) * rpg;
  if ((cap_rows + 63) / 64 > 65535) return FQT1_ERR_UNSUPPORTED;
  cudaStream_t s = (cudaStream_t)stream;
  if (!acc) {
    // dequantization fused into the tensor-core epilogue; pruned rows written as zeros
    FQT1_CUDA_TRY(launch_codes_tc_simple(p->bits, psq->codes, psq->ld_codes, cap_rows, psq->kept_count, rpg, sw_col,
                                         K, D, GEMM_EPI_DX, 1, nullptr, dx, K, psq->kept_idx, psq->scale,
                                         psq->zero, colsum_w, rpg, nullptr, s));
    launch_zero_pruned_rows(psq->slot_of_group, M, K, rpg, dx, s);
    FQT1_CUDA_TRY(cudaGetLastError());
    return FQT1_OK;
  }
  FQT1_CUDA_TRY(launch_codes_tc_simple(p->bits, psq->codes, psq->ld_codes, cap_rows, psq->kept_count, rpg, sw_col,
                                       K, D, GEMM_EPI_ACC32, 1, acc, nullptr, K, nullptr, nullptr, nullptr,
                                       nullptr, rpg, nullptr, s));
  if (dx) {
    const int64_t n = M * K;
    launch_k(dequant_rows_kernel, dim3((unsigned)((n + 255) / 256)), dim3(256), 0, s, acc, K, psq->slot_of_group, psq->scale,
                                                                    psq->zero, colsum_w, M, K, rpg, dx);
    fqt1_count_launches(1);
    FQT1_CUDA_TRY(cudaGetLastError());
  }
  return FQT1_OK;
}

// Words of a Folder CTA's tables after its accumulator tile: tap lists of hb rows and wb columns
// (offsets, column-sum offsets, counts) and the column sums of cb channels.
static int64_t fold_table_words(int64_t hb, int64_t wb, int64_t kh, int64_t kw, int64_t cb) {
  return 2 * hb * kh + hb + 2 * wb * kw + wb + cb * kh * kw;
}

// nhwc: dx in memory order N, H, W, C; only the tiled Folder writes it (else FQT1_ERR_UNSUPPORTED).
static fqt1_status col2im_impl(const int32_t* acc, const fqt1_qgrad* psq, const int32_t* colsum_w, int32_t N,
                               int32_t C, int32_t H, int32_t W, int32_t kh, int32_t kw, int32_t stride, int32_t pad,
                               float* dx, int nhwc, void* stream) {
  if (!acc || !psq || !colsum_w || !dx || N < 1 || C < 1 || H < 1 || W < 1 || kh < 1 || kw < 1 || stride < 1 ||
      pad < 0)
    return FQT1_ERR_INVALID_ARG;
  if (!psq->slot_of_group || !psq->scale || !psq->zero || !psq->kept_idx || !psq->kept_count)
    return FQT1_ERR_INVALID_ARG;
  const int64_t Ho64 = conv_extent(H, kh, stride, pad), Wo64 = conv_extent(W, kw, stride, pad);
  if (Ho64 == 0 || Wo64 == 0) return FQT1_ERR_INVALID_ARG;
  if (Ho64 < 0 || Wo64 < 0 || Ho64 * Wo64 >= (1ll << 31)) return FQT1_ERR_UNSUPPORTED;
  const int Ho = (int)Ho64, Wo = (int)Wo64;
  if (!aligned16(acc) || !aligned16(dx)) return FQT1_ERR_MISALIGNED;
  constexpr int64_t kMaxTile = 96 * 1024;
  constexpr int64_t kPreferTile = 48 * 1024;  // >= 4 resident CTAs per SM
  const int khw = kh * kw;
  if (kh == 1 && kw == 1 && pad == 0 && Wo <= 256 && (int64_t)Ho * ((C + 31) / 32) <= 0x7FFFFFFF && N <= 65535) {
    // pointwise convolution: one output row of 32 channels per CTA
    FoldArgs fa{};
    fa.acc = acc; fa.kept_idx = psq->kept_idx; fa.kept_count = psq->kept_count; fa.scale = psq->scale;
    fa.zero = psq->zero; fa.cs = colsum_w; fa.dx = dx; fa.N = N; fa.C = C; fa.H = H; fa.W = W; fa.kh = 1; fa.kw = 1;
    fa.stride = stride; fa.pad = 0; fa.Ho = Ho; fa.Wo = Wo; fa.K = C; fa.nhwc = nhwc;
    launch_zero_pruned_rows(psq->slot_of_group, N, (int64_t)C * H * W, 1, dx, (cudaStream_t)stream);
    const size_t smem = (size_t)32 * (Wo + 1) * 4;
    launch_k(col2im_pointwise_kernel, dim3((unsigned)((int64_t)Ho * ((C + 31) / 32)), (unsigned)N), dim3(256), smem,
             (cudaStream_t)stream, fa);
    fqt1_count_launches(1);
    FQT1_CUDA_TRY(cudaGetLastError());
    return FQT1_OK;
  }
  // whole-row Folder: up to 8 input rows per CTA and the most channels whose staged
  // accumulators fit (<= 48 KB, or 96 KB for a single channel)
  int hb = H < 8 ? H : 8, wb = W, cb = 0;
  int max_rows = 0, max_cols = Wo, kstride = 0;
  for (; hb >= 1 && cb == 0; hb /= 2) {
    max_rows = std::min(Ho, (hb - 1 + kh - 1) / stride + 1);
    for (int c = (C < 32 ? C : 32); c >= 1; c = (c > 1 ? c / 2 : 0)) {
      const int ks = (c * khw) | 1;
      const int64_t words = (int64_t)max_rows * Wo * ks + fold_table_words(hb, W, kh, kw, c);
      if (words * 4 <= (c > 1 ? kPreferTile : kMaxTile)) { cb = c; kstride = ks; break; }
    }
    if (cb) break;
  }
  // blocks of rows and columns when whole rows leave fewer than min(C, 4) channels per CTA:
  // chosen for the least staging cost per output (the halo of the windows and the partial
  // 32-byte sectors of each pixel's k-range, plus a fixed cost per CTA), with about 16 CTAs
  // per SM over all samples
  bool tiled = false;
  if (cb < std::min(C, 4)) {
    double best = 0.0;
    int tcb = 0;
    const int hbs[6] = {32, 16, 8, 4, 2, 1}, wbs[5] = {0, 64, 32, 16, 8};  // wb 0: whole rows
    for (int pass = 0; pass < 2 && tcb == 0; ++pass) {
      const int64_t cap = pass == 0 ? kPreferTile : kMaxTile;
      for (int hi = 0; hi < 6; ++hi) {
        const int hbc = hbs[hi] < H ? hbs[hi] : H;
        for (int wi = 0; wi < 5; ++wi) {
          const int wbc = (wbs[wi] == 0 || wbs[wi] > W) ? W : wbs[wi];
          const int mr = std::min(Ho, (hbc - 1 + kh - 1) / stride + 1);
          const int mc = std::min(Wo, (wbc - 1 + kw - 1) / stride + 1);
          for (int c = (C < 32 ? C : 32); c >= 1; c = (c > 1 ? c / 2 : 0)) {
            const int ks = (c * khw) | 1;
            const int64_t words = (int64_t)mr * mc * ks + fold_table_words(hbc, wbc, kh, kw, c);
            if (words * 4 > cap) continue;
            if ((int64_t)mr * Wo * C * khw >= (1ll << 31)) continue;  // the kernel's 32-bit halo offsets
            const double sectors = (double)(((int64_t)c * khw * 4 + 31) / 32 + 1) * 32.0;
            double cost = ((double)mr * mc * sectors + 8192.0) / ((double)hbc * wbc * c);
            const double ctas = (double)N * ((C + c - 1) / c) * ((H + hbc - 1) / hbc) * ((W + wbc - 1) / wbc);
            if (ctas < 16.0 * 152) cost *= 16.0 * 152 / ctas;
            if (tcb == 0 || cost < best) {
              best = cost; hb = hbc; wb = wbc; tcb = c; max_rows = mr; max_cols = mc; kstride = ks;
            }
          }
        }
      }
    }
    if (tcb > 0) { cb = tcb; tiled = true; }
  }
  if (cb > 0) {
    static std::atomic<uint64_t> attr_rows{0}, attr_tiled{0};
    FQT1_CUDA_TRY(smem_attr_once((const void*)col2im_rows_kernel, (int)kMaxTile, attr_rows));
    FQT1_CUDA_TRY(smem_attr_once((const void*)col2im_tiled_kernel, (int)kMaxTile, attr_tiled));
    FoldArgs fa;
    fa.acc = acc; fa.kept_idx = psq->kept_idx; fa.kept_count = psq->kept_count; fa.scale = psq->scale;
    fa.zero = psq->zero;
    fa.cs = colsum_w; fa.dx = dx; fa.N = N; fa.C = C; fa.H = H; fa.W = W; fa.kh = kh; fa.kw = kw;
    fa.stride = stride; fa.pad = pad; fa.Ho = Ho; fa.Wo = Wo; fa.cb = cb; fa.hb = hb; fa.wb = wb;
    fa.ncb = (C + cb - 1) / cb; fa.nwb = (W + wb - 1) / wb; fa.max_rows = max_rows; fa.max_cols = max_cols;
    fa.kstride = kstride; fa.K = (int64_t)C * khw;
    fa.nhwc = nhwc;
    const int64_t nblk = (int64_t)fa.ncb * fa.nwb * ((H + hb - 1) / hb);
    if (nblk > 0x7FFFFFFF || N > 65535) return FQT1_ERR_UNSUPPORTED;
    const size_t smem = ((size_t)max_rows * max_cols * kstride + (size_t)fold_table_words(hb, wb, kh, kw, cb)) * 4;
    // pruned samples: zeros; kept samples: the tiled fold (one grid row per kept slot)
    launch_zero_pruned_rows(psq->slot_of_group, N, (int64_t)C * H * W, 1, dx, (cudaStream_t)stream);
    const int64_t cap = fqt1_kept_capacity(N, 8, FQT1_SEL_BERNOULLI);  // upper bound: all samples
    launch_k(tiled ? col2im_tiled_kernel : col2im_rows_kernel, dim3((unsigned)nblk, (unsigned)cap), dim3(256), smem,
             (cudaStream_t)stream, fa);
  } else {
    if (nhwc) return FQT1_ERR_UNSUPPORTED;
    const int64_t n = (int64_t)N * C * H * W;
    launch_k(col2im_kernel, dim3((unsigned)((n + 255) / 256)), dim3(256), 0, (cudaStream_t)stream, 
        acc, psq->slot_of_group, psq->scale, psq->zero, colsum_w, N, C, H, W, kh, kw, stride, pad, Ho, Wo, dx);
  }
  fqt1_count_launches(1);
  FQT1_CUDA_TRY(cudaGetLastError());
  return FQT1_OK;
}

extern "C" fqt1_status fqt1_col2im(const int32_t* acc, const fqt1_qgrad* psq, const int32_t* colsum_w, int32_t N,
                                   int32_t C, int32_t H, int32_t W, int32_t kh, int32_t kw, int32_t stride,
                                   int32_t pad, float* dx, void* stream) {
  return col2im_impl(acc, psq, colsum_w, N, C, H, W, kh, kw, stride, pad, dx, 0, stream);
}

static fqt1_status bwd_input_colmajor_impl(const fqt1_qgrad* psq, const uint32_t* sw_col, const uint8_t* wt_e4m3,
                                           int64_t ld_wt, int64_t M, int64_t D, int64_t K, const fqt1_agp_params* p,
                                           void* acc, int32_t acc_bits, int64_t ld_acc, void* stream) {
  if (!psq || !(sw_col || wt_e4m3) || !p || !acc || M < 1 || D < 1 || K < 1) return FQT1_ERR_INVALID_ARG;
  if (acc_bits != 16 && acc_bits != 32) return FQT1_ERR_INVALID_ARG;
  if (wt_e4m3 && (ld_wt < fqt1_codes_ld(D) || ld_wt % 16)) return FQT1_ERR_INVALID_ARG;
  if (!valid_bits(p->bits) || p->rows_per_group < 1 || M % p->rows_per_group) return FQT1_ERR_INVALID_ARG;
  if (!psq->codes || !psq->kept_count || psq->ld_codes < fqt1_codes_ld(D) || psq->ld_codes % 16)
    return FQT1_ERR_INVALID_ARG;
  const int64_t rpg = p->rows_per_group;
  const int64_t cap_rows = fqt1_kept_capacity(M / rpg, p->bits, p->mode) * rpg;
  if (ld_acc < cap_rows || ld_acc % (acc_bits == 16 ? 8 : 4)) return FQT1_ERR_INVALID_ARG;
  // int16 sums: every |acc| <= (2^b - 1) D must fit
  if (acc_bits == 16 && ((1ll << p->bits) - 1) * D > 32767) return FQT1_ERR_INVALID_ARG;
  if ((sw_col && !aligned16(sw_col)) || (wt_e4m3 && !aligned16(wt_e4m3)) || !aligned16(acc))
    return FQT1_ERR_MISALIGNED;
  if ((cap_rows + 63) / 64 > 65535) return FQT1_ERR_UNSUPPORTED;
  FQT1_CUDA_TRY(launch_codes_tc_colmajor(p->bits, psq->codes, psq->ld_codes, cap_rows, psq->kept_count, rpg, sw_col,
                                         K, D, acc, acc_bits, ld_acc, nullptr, (cudaStream_t)stream, wt_e4m3, ld_wt));
  return FQT1_OK;
}

extern "C" fqt1_status fqt1_bwd_input_gemm_colmajor(const fqt1_qgrad* psq, const uint32_t* sw_col, int64_t M,
                                                    int64_t D, int64_t K, const fqt1_agp_params* p, void* acc,
                                                    int32_t acc_bits, int64_t ld_acc, void* stream) {
  if (!sw_col) return FQT1_ERR_INVALID_ARG;
  return bwd_input_colmajor_impl(psq, sw_col, nullptr, 0, M, D, K, p, acc, acc_bits, ld_acc, stream);
}

extern "C" fqt1_status fqt1_bwd_input_gemm_colmajor_e4m3w(const fqt1_qgrad* psq, const uint8_t* wt_e4m3, int64_t ld_wt,
                                                          int64_t M, int64_t D, int64_t K, const fqt1_agp_params* p,
                                                          void* acc, int32_t acc_bits, int64_t ld_acc, void* stream) {
  if (!wt_e4m3) return FQT1_ERR_INVALID_ARG;
  return bwd_input_colmajor_impl(psq, nullptr, wt_e4m3, ld_wt, M, D, K, p, acc, acc_bits, ld_acc, stream);
}

static fqt1_status col2im_colmajor_impl(const void* acc, int32_t acc_bits, int64_t ld_acc, const fqt1_qgrad* psq,
                                       const int32_t* colsum_w, int32_t N, int32_t C, int32_t H, int32_t W,
                                       int32_t kh, int32_t kw, int32_t stride, int32_t pad, float* dx, bool nhwc,
                                       void* stream) {
  if (!acc || !psq || !colsum_w || !dx || N < 1 || C < 1 || H < 1 || W < 1 || kh < 1 || kw < 1 || stride < 1 ||
      pad < 0 || kh > 64 || kw > 64)
    return FQT1_ERR_INVALID_ARG;
  if (!psq->slot_of_group || !psq->scale || !psq->zero || !psq->kept_idx || !psq->kept_count)
    return FQT1_ERR_INVALID_ARG;
  const int64_t Ho64 = conv_extent(H, kh, stride, pad), Wo64 = conv_extent(W, kw, stride, pad);
  if (Ho64 == 0 || Wo64 == 0) return FQT1_ERR_INVALID_ARG;
  if (Ho64 < 0 || Wo64 < 0 || Ho64 * Wo64 >= (1ll << 31)) return FQT1_ERR_UNSUPPORTED;
  const int Ho = (int)Ho64, Wo = (int)Wo64;
  if (acc_bits != 16 && acc_bits != 32) return FQT1_ERR_INVALID_ARG;
  if (ld_acc < (int64_t)Ho * Wo || ld_acc % (acc_bits == 16 ? 8 : 4)) return FQT1_ERR_INVALID_ARG;
  if (!aligned16(acc) || !aligned16(dx)) return FQT1_ERR_MISALIGNED;
  const int64_t plane = (int64_t)C * H * W;
  if (plane >= (1ll << 31) || N > 65535) return FQT1_ERR_UNSUPPORTED;
  FoldCmArgs fa;
  fa.acc = acc; fa.ld = ld_acc; fa.kept_idx = psq->kept_idx; fa.kept_count = psq->kept_count;
  fa.scale = psq->scale; fa.zero = psq->zero; fa.cs = colsum_w; fa.dx = dx;
  fa.H = H; fa.W = W; fa.kh = kh; fa.kw = kw; fa.stride = stride; fa.pad = pad; fa.Ho = Ho; fa.Wo = Wo;
  fa.plane = plane; fa.div_hw = FastDiv((uint32_t)(H * W)); fa.div_w = FastDiv((uint32_t)W);
  const int64_t K = (int64_t)C * kh * kw;
  if (K >= (1ll << 31)) return FQT1_ERR_UNSUPPORTED;  // column indices are 32-bit in the kernels
  fa.K = (int)K;
  fa.cs_smem = K <= 12288;
  const size_t cs_bytes = fa.cs_smem ? (size_t)K * 4 : 0;
  cudaStream_t s = (cudaStream_t)stream;
  // pruned samples: zeros; kept samples: one grid row per slot (slots past the kept count exit)
  launch_zero_pruned_rows(psq->slot_of_group, N, plane, 1, dx, s);
  // grid: the plane's CTAs along x; along y about 16 CTAs per SM in all (a few resident waves),
  // each grid row looping over kept slots y, y + gridDim.y, ...
  auto grid = [&](int per) {
    const int64_t gx = (plane + 256 * per - 1) / (256 * per);
    const int64_t gy = std::max<int64_t>(1, std::min<int64_t>(N, (16 * (int64_t)sm_count_api() + gx - 1) / gx));
    return dim3((unsigned)gx, (unsigned)gy);
  };
  if (nhwc) {  // 32 positions x 32 channels per CTA, the same grid rows over kept slots
    const int64_t gx = ((int64_t)H * W + 31) / 32 * ((C + 31) / 32);
    if (gx > 0x7FFFFFFF) return FQT1_ERR_UNSUPPORTED;
    const dim3 g((unsigned)gx,
                 (unsigned)std::max<int64_t>(1, std::min<int64_t>(N, (16 * (int64_t)sm_count_api() + gx - 1) / gx)));
    auto launch_nhwc = [&](auto zero) {
      using T = decltype(zero);
      if (kh == 3 && kw == 3 && stride == 1)
        launch_k(col2im_colmajor_nhwc_kernel<3, 3, 1, T>, g, dim3(256), cs_bytes, s, fa);
      else if (kh == 3 && kw == 3 && stride == 2)
        launch_k(col2im_colmajor_nhwc_kernel<3, 3, 2, T>, g, dim3(256), cs_bytes, s, fa);
      else if (kh == 1 && kw == 1 && stride == 1)
        launch_k(col2im_colmajor_nhwc_kernel<1, 1, 1, T>, g, dim3(256), cs_bytes, s, fa);
      else if (kh == 1 && kw == 1 && stride == 2)
        launch_k(col2im_colmajor_nhwc_kernel<1, 1, 2, T>, g, dim3(256), cs_bytes, s, fa);
      else
        launch_k(col2im_colmajor_nhwc_kernel<0, 0, 0, T>, g, dim3(256), cs_bytes, s, fa);
    };
    if (acc_bits == 16)
      launch_nhwc(int16_t{0});
    else
      launch_nhwc(int32_t{0});
    fqt1_count_launches(1);
    FQT1_CUDA_TRY(cudaGetLastError());
    return FQT1_OK;
  }
  auto launch = [&](auto zero) {  // zero: a value of the accumulator type
    using T = decltype(zero);
    if (kh == 3 && kw == 3 && stride == 1)
      launch_k(col2im_colmajor_kernel<3, 3, 1, T>, grid(fold_cm_per(3, 3, 1)), dim3(256), cs_bytes, s, fa);
    else if (kh == 3 && kw == 3 && stride == 2)
      launch_k(col2im_colmajor_kernel<3, 3, 2, T>, grid(fold_cm_per(3, 3, 2)), dim3(256), cs_bytes, s, fa);
    else if (kh == 1 && kw == 1 && stride == 1)
      launch_k(col2im_colmajor_kernel<1, 1, 1, T>, grid(fold_cm_per(1, 1, 1)), dim3(256), cs_bytes, s, fa);
    else if (kh == 1 && kw == 1 && stride == 2)
      launch_k(col2im_colmajor_kernel<1, 1, 2, T>, grid(fold_cm_per(1, 1, 2)), dim3(256), cs_bytes, s, fa);
    else if (kh == 7 && kw == 7 && stride == 2)
      launch_k(col2im_colmajor_kernel<7, 7, 2, T>, grid(fold_cm_per(7, 7, 2)), dim3(256), cs_bytes, s, fa);
    else
      launch_k(col2im_colmajor_kernel<0, 0, 0, T>, grid(fold_cm_per(0, 0, 1)), dim3(256), cs_bytes, s, fa);
  };
  if (acc_bits == 16)
    launch(int16_t{0});
  else
    launch(int32_t{0});
  fqt1_count_launches(1);
  FQT1_CUDA_TRY(cudaGetLastError());
  return FQT1_OK;
}

extern "C" fqt1_status fqt1_col2im_colmajor(const void* acc, int32_t acc_bits, int64_t ld_acc, const fqt1_qgrad* psq,
                                            const int32_t* colsum_w, int32_t N, int32_t C, int32_t H, int32_t W,
                                            int32_t kh, int32_t kw, int32_t stride, int32_t pad, float* dx,
                                            void* stream) {
  return col2im_colmajor_impl(acc, acc_bits, ld_acc, psq, colsum_w, N, C, H, W, kh, kw, stride, pad, dx, false,
                              stream);
}

extern "C" fqt1_status fqt1_col2im_colmajor_nhwc(const void* acc, int32_t acc_bits, int64_t ld_acc,
                                                 const fqt1_qgrad* psq, const int32_t* colsum_w, int32_t N,
                                                 int32_t C, int32_t H, int32_t W, int32_t kh, int32_t kw,
                                                 int32_t stride, int32_t pad, float* dx, void* stream) {
  return col2im_colmajor_impl(acc, acc_bits, ld_acc, psq, colsum_w, N, C, H, W, kh, kw, stride, pad, dx, true,
                              stream);
}

extern "C" fqt1_status fqt1_col2im_nhwc(const int32_t* acc, const fqt1_qgrad* psq, const int32_t* colsum_w, int32_t N,
                                        int32_t C, int32_t H, int32_t W, int32_t kh, int32_t kw, int32_t stride,
                                        int32_t pad, float* dx, void* stream) {
  return col2im_impl(acc, psq, colsum_w, N, C, H, W, kh, kw, stride, pad, dx, 1, stream);
}

// Shared by the two Folder entry points: B is the packed sign(W) columns sw_col, or (wt_e4m3
// non-null) the e4m3 bytes of sign(W)^T with rows of ld_wt bytes.
static fqt1_status bwd_input_fold_impl(const fqt1_qgrad* psq, const uint32_t* sw_col, const uint8_t* wt_e4m3,
                                       int64_t ld_wt, const int32_t* colsum_w, int32_t N, int32_t C, int32_t H,
                                       int32_t W, int32_t kh, int32_t kw, int32_t stride, int32_t pad, int64_t D,
                                       const fqt1_agp_params* p, float* dx, int nhwc, void* stream) {
  if (!psq || (!sw_col && !wt_e4m3) || !colsum_w || !p || !dx || N < 1 || C < 1 || H < 1 || W < 1 || kh < 1 ||
      kw < 1 || stride < 1 || pad < 0 || D < 1)
    return FQT1_ERR_INVALID_ARG;
  if (wt_e4m3 && (ld_wt < D || ld_wt % 16)) return FQT1_ERR_INVALID_ARG;
  if (wt_e4m3 && !aligned16(wt_e4m3)) return FQT1_ERR_MISALIGNED;
  if (!valid_bits(p->bits) || !psq->codes || !psq->kept_count || !psq->kept_idx || !psq->slot_of_group ||
      !psq->scale || !psq->zero || psq->ld_codes < fqt1_codes_ld(D) || psq->ld_codes % 16)
    return FQT1_ERR_INVALID_ARG;
  const int64_t Ho64 = conv_extent(H, kh, stride, pad), Wo64 = conv_extent(W, kw, stride, pad);
  if (Ho64 == 0 || Wo64 == 0) return FQT1_ERR_INVALID_ARG;
  if (Ho64 < 0 || Wo64 < 0 || Ho64 * Wo64 >= (1ll << 31)) return FQT1_ERR_UNSUPPORTED;
  const int Ho = (int)Ho64, Wo = (int)Wo64;
  if (p->rows_per_group != (int64_t)Ho * Wo) return FQT1_ERR_INVALID_ARG;
  if ((sw_col && !aligned16(sw_col)) || !aligned16(dx) || !aligned16(colsum_w)) return FQT1_ERR_MISALIGNED;
  // whole samples per 128-row tile, at least one channel's taps per tile, and the Folder's
  // tables (tap offsets, folded colsums of 128 / (kh kw) channels, per-sample constants) in
  // their 36 KB of shared memory
  if (128 % (Ho * Wo) != 0 || kh * kw > 128 || fold_table_bytes(H, W, kh, kw, Ho, Wo) > 36864 ||
      (int64_t)N * C * H * W >= (1ll << 31))
    return FQT1_ERR_UNSUPPORTED;
  cudaStream_t s = (cudaStream_t)stream;
  const int64_t rpg = (int64_t)Ho * Wo;
  const int64_t cap_rows = fqt1_kept_capacity(N, p->bits, p->mode) * rpg;
  FQT1_CUDA_TRY(launch_fold_tc(p->bits, psq->codes, psq->ld_codes, cap_rows, psq->kept_count, sw_col,
                               (int64_t)C * kh * kw, D, psq->kept_idx, psq->scale, psq->zero, colsum_w,
                               psq->slot_of_group, dx, N, C, H, W, kh, kw, stride, pad, Ho, Wo, nullptr, s,
                               wt_e4m3, ld_wt, nhwc));
  return FQT1_OK;
}

extern "C" fqt1_status fqt1_bwd_input_fold(const fqt1_qgrad* psq, const uint32_t* sw_col, const int32_t* colsum_w,
                                           int32_t N, int32_t C, int32_t H, int32_t W, int32_t kh, int32_t kw,
                                           int32_t stride, int32_t pad, int64_t D, const fqt1_agp_params* p,
                                           float* dx, void* stream) {
  if (!sw_col) return FQT1_ERR_INVALID_ARG;
  return bwd_input_fold_impl(psq, sw_col, nullptr, 0, colsum_w, N, C, H, W, kh, kw, stride, pad, D, p, dx, 0, stream);
}

extern "C" fqt1_status fqt1_bwd_input_fold_nhwc(const fqt1_qgrad* psq, const uint32_t* sw_col,
                                                const int32_t* colsum_w, int32_t N, int32_t C, int32_t H, int32_t W,
                                                int32_t kh, int32_t kw, int32_t stride, int32_t pad, int64_t D,
                                                const fqt1_agp_params* p, float* dx, void* stream) {
  if (!sw_col) return FQT1_ERR_INVALID_ARG;
  return bwd_input_fold_impl(psq, sw_col, nullptr, 0, colsum_w, N, C, H, W, kh, kw, stride, pad, D, p, dx, 1, stream);
}

extern "C" fqt1_status fqt1_bwd_input_fold_e4m3w(const fqt1_qgrad* psq, const uint8_t* wt_e4m3, int64_t ld_wt,
                                                 const int32_t* colsum_w, int32_t N, int32_t C, int32_t H, int32_t W,
                                                 int32_t kh, int32_t kw, int32_t stride, int32_t pad, int64_t D,
                                                 const fqt1_agp_params* p, float* dx, void* stream) {
  if (!wt_e4m3) return FQT1_ERR_INVALID_ARG;
  return bwd_input_fold_impl(psq, nullptr, wt_e4m3, ld_wt, colsum_w, N, C, H, W, kh, kw, stride, pad, D, p, dx,
                             0, stream);
}

// grad_weight with B = packed sign(X_u)^T words (sx_col) or e4m3 sign bytes (xe, ldxe).
static fqt1_status bwd_weight_impl(const fqt1_qgrad* pcq, const uint32_t* sx_col, const uint8_t* xe, int64_t ldxe,
                                   const int32_t* colsum_x, int64_t M, int64_t D, int64_t K,
                                   const fqt1_agp_params* p, int32_t* acc, float* dw, void* stream) {
  if (!pcq || (!sx_col && !xe) || !colsum_x || !p || !acc || !dw || M < 1 || D < 1 || K < 1)
    return FQT1_ERR_INVALID_ARG;
  if (!valid_bits(p->bits)) return FQT1_ERR_INVALID_ARG;
  if (!pcq->codes || !pcq->kept_count || !pcq->slot_of_group || !pcq->scale || !pcq->zero ||
      pcq->ld_codes < fqt1_codes_ld(M) || pcq->ld_codes % 16)
    return FQT1_ERR_INVALID_ARG;
  if (xe && (ldxe < fqt1_codes_ld(M) || ldxe % 16)) return FQT1_ERR_INVALID_ARG;
  if ((sx_col && !aligned16(sx_col)) || (xe && !aligned16(xe)) || !aligned16(acc) || !aligned16(dw) ||
      !aligned16(colsum_x))
    return FQT1_ERR_MISALIGNED;
  const int64_t cap = fqt1_kept_capacity(D, p->bits, p->mode);
  cudaStream_t s = (cudaStream_t)stream;
  {
    // split the long contraction over M across a cluster of CTAs that reduce their int32
    // partial tiles in shared memory and dequantize in the same kernel; each CTA's fp32 partial
    // sum stays below 2^24 and no split is empty (every CTA of a cluster takes part)
    const int64_t k_tiles = (M + kCodesStageK - 1) / kCodesStageK;  // pipeline stages
    const int64_t out_tiles_c = ((K + 127) / 128) * ((cap + 127) / 128);
    int64_t cs = wgrad_cluster_size(p->bits, out_tiles_c, k_tiles);
    int64_t tps = (k_tiles + cs - 1) / cs;
    cs = (k_tiles + tps - 1) / tps;
    // few output tiles over a long contraction (e.g. 16 kept channels x 576 columns over 131072
    // rows) leave most SMs idle with clusters of at most 8 splits: the atomic reduction below then
    // spreads the contraction over about one wave of CTAs instead
    const int64_t red_splits = std::min<int64_t>(k_tiles, std::max<int64_t>((152 + out_tiles_c - 1) / out_tiles_c,
                                                                            (M + exact_chunk(p->bits) - 1) /
                                                                                exact_chunk(p->bits)));
    const bool spread = tps > 8 && red_splits >= 2 * cs;
    if (!spread && tps * kCodesStageK <= exact_chunk(p->bits)) {
      FQT1_CUDA_TRY(launch_wgrad_cluster_tc(p->bits, pcq->codes, pcq->ld_codes, cap, pcq->kept_count, sx_col, K, M,
                                            (int)cs, acc, dw, D, pcq->kept_idx, pcq->slot_of_group, pcq->scale,
                                            pcq->zero, colsum_x, nullptr, s, xe, ldxe));
      return FQT1_OK;
    }
    // contractions too long for eight exact splits, or too long for so few clusters: int32
    // atomics across CTAs, then dequantize
    const int64_t out_tiles = ((K + 127) / 128) * ((cap + 127) / 128);
    int64_t splits = (152 + out_tiles - 1) / out_tiles;  // about one wave on 152 SMs
    const int64_t min_splits = (M + exact_chunk(p->bits) - 1) / exact_chunk(p->bits);
    if (splits < min_splits) splits = min_splits;
    if (splits > k_tiles) splits = k_tiles;
    if ((k_tiles + splits - 1) / splits * kCodesStageK > exact_chunk(p->bits)) return FQT1_ERR_UNSUPPORTED;
    FQT1_CUDA_TRY(cudaMemsetAsync(acc, 0, sizeof(int32_t) * cap * K, s));
    FQT1_CUDA_TRY(launch_codes_tc_simple(p->bits, pcq->codes, pcq->ld_codes, cap, pcq->kept_count, 1, sx_col, K, M,
                                         GEMM_EPI_RED, (int)splits, acc, nullptr, K, nullptr, nullptr, nullptr,
                                         nullptr, 1, nullptr, s, xe, ldxe));
  }
  const int64_t n = D * K;
  launch_k(dequant_rows_kernel, dim3((unsigned)((n + 255) / 256)), dim3(256), 0, s, acc, K, pcq->slot_of_group, pcq->scale, pcq->zero,
                                                                  colsum_x, D, K, 1, dw);
  fqt1_count_launches(1);
  FQT1_CUDA_TRY(cudaGetLastError());
  return FQT1_OK;
}

extern "C" fqt1_status fqt1_bwd_weight_gemm(const fqt1_qgrad* pcq, const uint32_t* sx_col, const int32_t* colsum_x,
                                            int64_t M, int64_t D, int64_t K, const fqt1_agp_params* p, int32_t* acc,
                                            float* dw, void* ws, size_t ws_bytes, void* stream) {
  (void)ws; (void)ws_bytes;
  if (!sx_col) return FQT1_ERR_INVALID_ARG;
  return bwd_weight_impl(pcq, sx_col, nullptr, 0, colsum_x, M, D, K, p, acc, dw, stream);
}

extern "C" fqt1_status fqt1_bwd_weight_gemm_e4m3x(const fqt1_qgrad* pcq, const uint8_t* x_col_e4m3, int64_t ld_xc,
                                                  const int32_t* colsum_x, int64_t M, int64_t D, int64_t K,
                                                  const fqt1_agp_params* p, int32_t* acc, float* dw, void* stream) {
  if (!x_col_e4m3) return FQT1_ERR_INVALID_ARG;
  return bwd_weight_impl(pcq, nullptr, x_col_e4m3, ld_xc, colsum_x, M, D, K, p, acc, dw, stream);
}

extern "C" fqt1_status fqt1_fwd_gemm_e4m3x(const uint8_t* x_e4m3, int64_t ld_x, const uint8_t* w_e4m3, int64_t ld_w,
                                           int64_t M, int64_t D, int64_t K, const float* gamma, const float* bias,
                                           int32_t* acc, float* y, void* stream) {
  if (!x_e4m3 || !w_e4m3 || M < 1 || D < 1 || K < 1 || (!acc && !y) || (y && !gamma) || (bias && !y))
    return FQT1_ERR_INVALID_ARG;
  if (ld_x < fqt1_codes_ld(K) || ld_x % 16 || ld_w < fqt1_codes_ld(K) || ld_w % 16) return FQT1_ERR_INVALID_ARG;
  if (!aligned16(x_e4m3) || !aligned16(w_e4m3) || (acc && !aligned16(acc)) || (y && !aligned16(y)) ||
      (gamma && !aligned16(gamma)) || (bias && !aligned16(bias)))
    return FQT1_ERR_MISALIGNED;
  if (K >= (1ll << 24) || (M + 127) / 128 > 65535) return FQT1_ERR_UNSUPPORTED;
  FQT1_CUDA_TRY(launch_fwd_e4m3x_tc(x_e4m3, ld_x, w_e4m3, ld_w, M, D, K, gamma, bias, acc, y, nullptr,
                                    (cudaStream_t)stream));
  return FQT1_OK;
}

