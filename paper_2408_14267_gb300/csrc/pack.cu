// Sign + pack kernels: the row / column encoders of App. C (Algorithm 2) and the
// Unfolder fused with them.  One pass over the input writes both packings and
// the column sums of the signs.
#include <algorithm>

#include "common.cuh"

namespace fqt1 {

// A CTA covers Loader::kRows rows (32 or 64) x 256 columns (8 packed words) of the
// logical matrix.  Warp w packs rows w, w+8, ... along the columns with __ballot_sync;
// the row words of each 32-column slab then give, read bit-wise per column, the
// column-packed words of those rows (one per 32 rows).
constexpr int kPackWordsPerCta = 8;

// A loader splits element (r, c) into a per-row part and a per-column part, so that a
// warp computes its row part once per row and a lane its column parts once per CTA.  The
// gather path below serves unfolds whose input region does not fit the bit-level kernel.
// Element (m, k) of the unfolded matrix X_u = Unfolder(x); outside the image it is 0.
// Column k = (c*kh + i)*kw + j, row m = (n*Ho + oh)*Wo + ow.  All indices fit in 32 bits
// (checked on the host); divisions by the layer's constants use FastDiv.
struct Im2colLoader {
  static constexpr int kRows = 64;
  const float* x;
  int64_t rows, cols;  // M = N*Ho*Wo, K = C*kh*kw
  int H, W, stride, pad, CHW, HW;
  FastDiv div_hw_out, div_wo, div_khw, div_kw;
  struct Col { int off, i, j; bool ok; };
  struct Row { int base, h0, w0; bool ok; };
  __device__ __forceinline__ Col col(int64_t k64) const {
    Col o{0, 0, 0, k64 < cols};
    if (o.ok) {
      const uint32_t k = (uint32_t)k64;
      const uint32_t c = div_khw.div(k), t = k - c * div_khw.d;
      o.i = (int)div_kw.div(t);
      o.j = (int)(t - (uint32_t)o.i * div_kw.d);
      o.off = (int)c * HW;
    }
    return o;
  }
  __device__ __forceinline__ Row row(int64_t m64) const {
    Row o{0, 0, 0, m64 < rows};
    if (o.ok) {
      const uint32_t m = (uint32_t)m64;
      const uint32_t n = div_hw_out.div(m), rem = m - n * div_hw_out.d;
      const uint32_t oh = div_wo.div(rem), ow = rem - oh * div_wo.d;
      o.base = (int)n * CHW;
      o.h0 = (int)oh * stride - pad;
      o.w0 = (int)ow * stride - pad;
    }
    return o;
  }
  __device__ __forceinline__ float load(const Row& r, const Col& c) const {
    const int h = r.h0 + c.i, w = r.w0 + c.j;
    const bool in = r.ok && c.ok && (unsigned)h < (unsigned)H && (unsigned)w < (unsigned)W;
    return in ? __ldg(x + (r.base + c.off + h * W + w)) : 0.0f;
  }
};

template <class Loader>
__global__ void __launch_bounds__(256) pack_kernel(Loader L, uint32_t* __restrict__ row_bits, int64_t row_words,
                                                   uint32_t* __restrict__ col_bits, int64_t col_words,
                                                   int32_t* __restrict__ colsum) {
  FQT1_PDL_WAIT();
  FQT1_PDL_TRIGGER();
  constexpr int R = Loader::kRows;
  __shared__ uint32_t rw[R][kPackWordsPerCta];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t r0 = (int64_t)blockIdx.y * R;
  const int64_t w0 = (int64_t)blockIdx.x * kPackWordsPerCta;
  typename Loader::Col cols[kPackWordsPerCta];
#pragma unroll
  for (int q = 0; q < kPackWordsPerCta; ++q) cols[q] = L.col((w0 + q) * 32 + lane);
  // all loads of this warp's rows first, then the ballots
  float v[R / 8][kPackWordsPerCta];
#pragma unroll
  for (int i = 0; i < R / 8; ++i) {
    const typename Loader::Row row = L.row(r0 + warp + 8 * i);
#pragma unroll
    for (int q = 0; q < kPackWordsPerCta; ++q) v[i][q] = L.load(row, cols[q]);
  }
#pragma unroll
  for (int i = 0; i < R / 8; ++i) {
#pragma unroll
    for (int q = 0; q < kPackWordsPerCta; ++q) {
      const uint32_t word = __ballot_sync(0xFFFFFFFFu, v[i][q] > 0.0f);
      if (lane == 0) rw[warp + 8 * i][q] = word;
    }
  }
  __syncthreads();
  // Row-packed output: word (r, w0 + q).
  if (row_bits) {
    for (int e = threadIdx.x; e < R * kPackWordsPerCta; e += 256) {
      const int rr = e >> 3, q = e & 7;
      const int64_t r = r0 + rr, w = w0 + q;
      if (r < L.rows && w < row_words) row_bits[r * row_words + w] = rw[rr][q];
    }
  }
  // Column-packed output: word (c, r0/32 + h) holds rows r0+32h .. r0+32h+31 of column c.
  const int q = threadIdx.x >> 5;
  const int64_t c = (w0 + q) * 32 + lane;
  if (c < L.cols) {
    int sum = 0;
#pragma unroll
    for (int h = 0; h < R / 32; ++h) {
      uint32_t cw = 0;
#pragma unroll
      for (int rr = 0; rr < 32; ++rr) cw |= ((rw[32 * h + rr][q] >> lane) & 1u) << rr;
      const int64_t wi = r0 / 32 + h;
      if (col_bits && wi < col_words) col_bits[c * col_words + wi] = cw;
      const int64_t nvalid = min((int64_t)32, L.rows - (r0 + 32 * h));
      if (nvalid > 0) sum += 2 * __popc(cw) - (int)nvalid;
    }
    if (colsum) atomicAdd(colsum + c, sum);
  }
}

// Dense sign-pack: one warp per 32 x 32 block of x.  Lane l loads column c0 + l of the
// block's 32 rows (32 independent coalesced loads), forms that column's word with shifts,
// and the 32 ballots give the block's row words (lane i keeps row i's word).
__global__ void __launch_bounds__(128) pack_dense_kernel(const float* __restrict__ x, int64_t rows, int64_t cols,
                                                         int64_t ld, uint32_t* __restrict__ row_bits,
                                                         int64_t row_words, uint32_t* __restrict__ col_bits,
                                                         int64_t col_words, int32_t* __restrict__ colsum) {
  FQT1_PDL_WAIT();
  FQT1_PDL_TRIGGER();
  const int lane = threadIdx.x & 31;
  const int64_t wb = (int64_t)blockIdx.x * 4 + (threadIdx.x >> 5);  // word column of the block
  const int64_t rb = blockIdx.y;                                    // 32-row band
  if (wb >= row_words) return;
  const int64_t c = wb * 32 + lane, r0 = rb * 32;
  const bool cok = c < cols;
  // unconditional loads from clamped addresses (masked afterwards): all 32 are issued before
  // the first ballot instead of one dependent round trip per row
  const float* xc = x + min(c, cols - 1);
  float v[32];
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __ldg(xc + min(r0 + i, rows - 1) * ld);
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = (cok && r0 + i < rows) ? v[i] : 0.0f;
  uint32_t cw = 0, rw = 0;
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    const uint32_t bit = v[i] > 0.0f ? 1u : 0u;
    cw |= bit << i;
    const uint32_t b = __ballot_sync(0xFFFFFFFFu, bit);
    if (lane == i) rw = b;
  }
  if (row_bits && r0 + lane < rows) row_bits[(r0 + lane) * row_words + wb] = rw;
  if (cok) {
    if (col_bits) col_bits[c * col_words + rb] = cw;
    if (colsum) atomicAdd(colsum + c, 2 * __popc(cw) - (int)min((int64_t)32, rows - r0));
  }
}

// Column-packed words past ceil(rows/32) (the alignment padding) are zero.
__global__ void zero_col_pad_kernel(uint32_t* col_bits, int64_t cols, int64_t col_words, int64_t first_pad) {
  FQT1_PDL_WAIT();
  FQT1_PDL_TRIGGER();
  const int64_t npad = col_words - first_pad;
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i < cols * npad) col_bits[(i / npad) * col_words + first_pad + (i % npad)] = 0u;
}

// ---------------------------------------------------------------------------
// Bit-level Unfolder.  A CTA owns tm output pixels x 256 columns of X_u.
//  1. It sign-packs the part of the input those entries read into shared memory: for
//     every (image, channel) pair of the region, input rows h_lo..h_hi form one bit
//     stream (bit e = sign of the e-th float of those rows, behind one zero guard word
//     and followed by another).
//  2. Warp w builds the 32 x 32 bit blocks of columns k0 + 32 w .. + 31.  For stride 1
//     a lane builds the column word of one k (a run of output pixels on one output row
//     reads a run of consecutive stream bits); otherwise a lane builds the row word of
//     one pixel (a run of kernel taps on one input row reads consecutive stream bits).
//     A 5-step shuffle butterfly transposes each block into the other packing.
//  3. Row words and column words are staged in shared memory and written as 32-byte runs.
constexpr int kUnfoldMaxStreamWords = 24576;  // 96 KB of input bit streams per CTA

struct UnfoldArgs {
  const float* x;
  const uint32_t* planes;  // or the sign bits of x as planes [N][C][pw] words (then x is unused)
  int pw;                  // words per plane, ceil(H W / 32)
  uint32_t* row_bits;
  uint32_t* col_bits;
  int32_t* colsum;
  int64_t row_words, col_words;
  int C, H, W, kh, kw, stride, pad, Wo, M, K, khw, HWo;
  int tm;     // output pixels per CTA: 32, 64, 128 or 256
  int guard;  // zero words before and after every plane stream
  int same;   // stride 1, kh = kw = 2 pad + 1, Ho Wo a multiple of 32 (fast column words)
  FastDiv div_khw, div_kw, div_hwo, div_wo;
};

// 32 x 32 bit transpose across a warp: lane r holds row r (bit c = column c); afterwards
// lane c holds column c (bit r = row r).  Step j swaps the off-diagonal j x j blocks: the
// lower lane of a pair keeps the low block of every 2j-bit field (mask m) and takes the
// partner's low block moved up by j; the upper lane keeps the high blocks and takes the
// partner's high blocks moved down.  A rotation by +-j followed by one bit select does
// either (the bits that wrap around land in the half that is not taken).
__device__ __forceinline__ uint32_t warp_transpose32(uint32_t x, int lane) {
#pragma unroll
  for (int j = 16; j >= 1; j >>= 1) {
    const uint32_t m = j == 16 ? 0x0000FFFFu : j == 8 ? 0x00FF00FFu : j == 4 ? 0x0F0F0F0Fu : j == 2 ? 0x33333333u
                                                                                                      : 0x55555555u;
    const bool up = (lane & j) != 0;
    const uint32_t p = __shfl_xor_sync(0xFFFFFFFFu, x, j);
    const uint32_t r = __funnelshift_l(p, p, up ? 32 - j : j);
    const uint32_t take = up ? m : ~m;
    x = (x & ~take) | (r & take);
  }
  return x;
}

// Dense sign-pack through shared memory, for rows of a multiple of 4 floats: a CTA loads a
// 32-row x 128-column tile with coalesced 16-byte loads (8 per thread, all in flight), lane l
// of warp w forms the column word of column 32 w + l from shared memory, the warp transpose
// gives the row words, and the row words leave as 16-byte stores.
constexpr int kPackTileWarps = 4;

// e4m3 bytes of 4 sign bits (bit k of nib -> byte k): +1 = 0x38, -1 = 0xB8.
__device__ __forceinline__ uint32_t e4m3_signs4(uint32_t nib) {
  return ((nib & 15u) * 0x10204080u & 0x80808080u) ^ 0xB8B8B8B8u;
}

// Optional outputs: the e4m3 bytes of the signs, rows [rows][ld_re] (columns cols .. ld_re - 1
// zero) and columns [cols][ld_ce] (rows rows .. ld_ce - 1 zero).
__global__ void __launch_bounds__(32 * kPackTileWarps) pack_tile_kernel(
    const float* __restrict__ x, int64_t rows, int64_t cols, int64_t ld, uint32_t* __restrict__ row_bits,
    int64_t row_words, uint32_t* __restrict__ col_bits, int64_t col_words, int32_t* __restrict__ colsum,
    uint8_t* __restrict__ row_e4m3, int64_t ld_re, uint8_t* __restrict__ col_e4m3, int64_t ld_ce) {
  constexpr int NW = kPackTileWarps, TC = 32 * NW, F4 = TC / 4;
  FQT1_PDL_WAIT();
  FQT1_PDL_TRIGGER();
  __shared__ __align__(16) float t[32][TC];
  __shared__ __align__(16) uint32_t rws[32][NW];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t r0 = (int64_t)blockIdx.y * 32, cb = (int64_t)blockIdx.x * TC;
  float4 v[8];
#pragma unroll
  for (int k = 0; k < 8; ++k) {  // unconditional loads from clamped positions, masked below
    const int idx = threadIdx.x + 32 * NW * k, r = idx / F4, c4 = idx % F4;
    v[k] = __ldg(reinterpret_cast<const float4*>(x + min(r0 + r, rows - 1) * ld + min(cb + 4 * c4, cols - 4)));
  }
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    const int idx = threadIdx.x + 32 * NW * k, r = idx / F4, c4 = idx % F4;
    const int64_t c = cb + 4 * c4;
    float4 w = v[k];
    if (r0 + r >= rows) w = make_float4(0.f, 0.f, 0.f, 0.f);
    if (c + 0 >= cols) w.x = 0.f;
    if (c + 1 >= cols) w.y = 0.f;
    if (c + 2 >= cols) w.z = 0.f;
    if (c + 3 >= cols) w.w = 0.f;
    *reinterpret_cast<float4*>(&t[r][4 * c4]) = w;
  }
  __syncthreads();
  const int cl = 32 * warp + lane;
  uint32_t cw = 0;
#pragma unroll
  for (int r = 0; r < 32; ++r) cw |= (t[r][cl] > 0.0f ? 1u : 0u) << r;
  rws[lane][warp] = warp_transpose32(cw, lane);
  const int64_t c = cb + cl;
  if (c < cols) {
    if (col_bits) col_bits[c * col_words + blockIdx.y] = cw;
    if (colsum) atomicAdd(colsum + c, 2 * __popc(cw) - (int)min((int64_t)32, rows - r0));
    if (col_e4m3) {  // column c, rows r0 .. r0 + 31 (up to ld_ce): 32 bytes from the column word
      const int nvalid = (int)min((int64_t)32, rows - r0);
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        if (r0 + 16 * h >= ld_ce) break;
        uint32_t wv[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          uint32_t v = e4m3_signs4(cw >> (16 * h + 4 * q));
#pragma unroll
          for (int b = 0; b < 4; ++b)
            if (16 * h + 4 * q + b >= nvalid) v &= ~(0xFFu << (8 * b));
          wv[q] = v;
        }
        *reinterpret_cast<uint4*>(col_e4m3 + c * ld_ce + r0 + 16 * h) = make_uint4(wv[0], wv[1], wv[2], wv[3]);
      }
    }
  }
  if (row_e4m3) {  // rows r0 .. r0 + 31, columns cb .. cb + TC - 1 (up to ld_re): 16 bytes per thread
    for (int e = threadIdx.x; e < 32 * (TC / 16); e += 32 * NW) {
      const int r = e / (TC / 16), q16 = e % (TC / 16);
      const int64_t c0 = cb + 16 * q16;
      if (r0 + r >= rows || c0 >= ld_re) continue;
      uint32_t wv[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        uint32_t nib = 0;
#pragma unroll
        for (int b = 0; b < 4; ++b) nib |= (t[r][16 * q16 + 4 * q + b] > 0.0f ? 1u : 0u) << b;
        uint32_t v = e4m3_signs4(nib);
#pragma unroll
        for (int b = 0; b < 4; ++b)
          if (c0 + 4 * q + b >= cols) v &= ~(0xFFu << (8 * b));
        wv[q] = v;
      }
      *reinterpret_cast<uint4*>(row_e4m3 + (r0 + r) * ld_re + c0) = make_uint4(wv[0], wv[1], wv[2], wv[3]);
    }
  }
  __syncthreads();
  if (row_bits) {  // row r: words cb / 32 .. + NW - 1
    for (int e = threadIdx.x; e < 32 * (NW / 4); e += 32 * NW) {
      const int r = e / (NW / 4), h = e % (NW / 4);
      const int64_t w0 = cb / 32 + 4 * h;
      if (r0 + r < rows && w0 < row_words)
        *reinterpret_cast<uint4*>(row_bits + (r0 + r) * row_words + w0) = *reinterpret_cast<const uint4*>(&rws[r][4 * h]);
    }
  }
}

// cnt (1..32) bits of a stream starting at bit pos; the guard words keep both reads inside.
__device__ __forceinline__ uint32_t stream_bits(const uint32_t* st, int pos, int cnt) {
  const int w = pos >> 5, o = pos & 31;
  const uint64_t v = ((uint64_t)st[w + 1] << 32) | st[w];
  const uint32_t bits = (uint32_t)(v >> o);
  return cnt >= 32 ? bits : bits & ((1u << cnt) - 1u);
}

// The even bits of 32 bits, packed into the low 16 (bit 2 t -> bit t).
__device__ __forceinline__ uint32_t even_bits16(uint32_t x) {
  x &= 0x55555555u;
  x = (x | (x >> 1)) & 0x33333333u;
  x = (x | (x >> 2)) & 0x0F0F0F0Fu;
  x = (x | (x >> 4)) & 0x00FF00FFu;
  x = (x | (x >> 8)) & 0x0000FFFFu;
  return x;
}

// cnt (1..32) bits of a stream at bit positions pos, pos + 2, ..., pos + 2 (cnt - 1): only the
// words holding those bits are read (at most three), so the read stays inside the bits it needs.
__device__ __forceinline__ uint32_t stream_even_bits(const uint32_t* st, int pos, int cnt) {
  const int w = pos >> 5, o = pos & 31, last = (pos + 2 * cnt - 2) >> 5;
  const uint32_t x0 = st[w];
  const uint32_t x1 = last > w ? st[w + 1] : 0u;
  const uint32_t x2 = last > w + 1 ? st[w + 2] : 0u;
  const uint32_t lo = __funnelshift_r(x0, x1, o), hi = __funnelshift_r(x1, x2, o);
  const uint32_t bits = even_bits16(lo) | (even_bits16(hi) << 16);
  return cnt >= 32 ? bits : bits & ((1u << cnt) - 1u);
}

__global__ void __launch_bounds__(256) unfold_bits_kernel(UnfoldArgs a) {
  FQT1_PDL_WAIT();
  FQT1_PDL_TRIGGER();
  extern __shared__ uint32_t stream[];
  __shared__ uint32_t rw_s[256][9];  // row words [pixel in tile][k-word in tile]
  __shared__ uint32_t cw_s[256][9];  // column words [k in tile][pixel-word in tile]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int m0 = blockIdx.y * a.tm, m1 = min(a.M, m0 + a.tm);
  const int k0 = blockIdx.x * 256, k1 = min(a.K, k0 + 256);
  const int nsub = a.tm / 32;
  const bool have_k = k0 < a.K;
  // region of the input read by this tile
  int c_lo = 0, nc = 1, n_lo = 0, h_lo = 0, nrows = 0, plane_words = 2, nplanes = 0;
  if (have_k) {
    c_lo = (int)a.div_khw.div((uint32_t)k0);
    nc = (int)a.div_khw.div((uint32_t)(k1 - 1)) - c_lo + 1;
    n_lo = (int)a.div_hwo.div((uint32_t)m0);
    const int n_hi = (int)a.div_hwo.div((uint32_t)(m1 - 1));
    int h_hi = a.H - 1;
    if (n_lo == n_hi) {
      const int oh_lo = (int)a.div_wo.div((uint32_t)(m0 - n_lo * a.HWo));
      const int oh_hi = (int)a.div_wo.div((uint32_t)(m1 - 1 - n_lo * a.HWo));
      h_lo = max(0, oh_lo * a.stride - a.pad);
      h_hi = min(a.H - 1, oh_hi * a.stride - a.pad + a.kh - 1);
    }
    nrows = max(0, h_hi - h_lo + 1);
    plane_words = (nrows * a.W + 31) / 32 + 2 * a.guard;
    nplanes = (n_hi - n_lo + 1) * nc;
  }
  // 1. sign-pack the region: word f of the region (plane f / data_words, word f % data_words of
  //    it) is the ballot of 32 consecutive floats of one plane row run; a warp takes words
  //    warp, warp + 8, ... with 16 loads in flight per lane (unconditional, from clamped
  //    indices), so the region costs one memory round trip per 128 words, not one per plane
  const int plane_bits = nrows * a.W, data_words = plane_words - 2 * a.guard, gbits = 32 * a.guard;
  if (a.planes) {
    // the signs are given as plane bits: word q of a region plane is the 32 bits from bit
    // h_lo W + 32 q of the full plane (a funnel shift of two words), zero past its rows
    // 8 region words per thread per batch, their 16 loads in flight together (unconditional,
    // from clamped indices)
    const int total = nplanes * data_words, bit0 = h_lo * a.W;
    const FastDiv div_dw((uint32_t)max(data_words, 1)), div_nc((uint32_t)nc);
    for (int f0 = threadIdx.x; f0 < total; f0 += 256 * 8) {
      uint32_t lo[8], hi[8];
      int pos[8], sh[8], left[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int f = min(f0 + 256 * u, total - 1);
        const int pl = (int)div_dw.div((uint32_t)f), q = f - pl * data_words;
        const int nn = (int)div_nc.div((uint32_t)pl), c = pl - nn * nc;
        const uint32_t* src = a.planes + ((int64_t)(n_lo + nn) * a.C + c_lo + c) * a.pw;
        const int b = bit0 + 32 * q, w0 = b >> 5;
        lo[u] = __ldg(src + min(w0, a.pw - 1));
        hi[u] = __ldg(src + min(w0 + 1, a.pw - 1));
        pos[u] = pl * plane_words + a.guard + q;
        sh[u] = b & 31;
        left[u] = plane_bits - 32 * q;
      }
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        if (f0 + 256 * u >= total) break;
        uint32_t word = __funnelshift_r(lo[u], hi[u], sh[u]);
        if (left[u] < 32) word &= left[u] <= 0 ? 0u : ((1u << left[u]) - 1u);
        stream[pos[u]] = word;
      }
    }
  } else if (nrows == a.H && plane_bits < 32 && 32 % plane_bits == 0) {  // plane_bits = H W >= 1 here
    // whole planes of fewer than 32 pixels that divide 32 (4 x 4, 2 x 2 maps): the region's
    // floats of one image are nc H W consecutive floats of x, so one ballot of 32 of them gives
    // the (single) words of 32 / (H W) consecutive planes; no load lane is idle
    const int hw = plane_bits, per = 32 / hw;
    const uint32_t pmask = (1u << hw) - 1u;
    const int span = nc * hw, gper = (span + 31) / 32;  // floats and ballots of one image's region
    const int total = (nplanes / nc) * gper;
    const int64_t img_stride = (int64_t)a.C * hw;
    const float* base = a.x + ((int64_t)n_lo * a.C + c_lo) * hw;
    const FastDiv div_g((uint32_t)gper);
    for (int f0 = warp; f0 < total; f0 += 8 * 16) {
      float v[16];
#pragma unroll
      for (int u = 0; u < 16; ++u) {
        const int f = min(f0 + 8 * u, total - 1);
        const int nn = (int)div_g.div((uint32_t)f), e = 32 * (f - nn * gper) + lane;
        v[u] = __ldg(base + nn * img_stride + min(e, span - 1));
        if (e >= span) v[u] = 0.0f;
      }
#pragma unroll
      for (int u = 0; u < 16; ++u) {
        const uint32_t word = __ballot_sync(0xFFFFFFFFu, v[u] > 0.0f);
        const int f = f0 + 8 * u;
        if (f < total && lane < per) {
          const int nn = (int)div_g.div((uint32_t)f), c = (f - nn * gper) * per + lane;
          if (c < nc) stream[(nn * nc + c) * plane_words + a.guard] = (word >> (lane * hw)) & pmask;
        }
      }
    }
  } else {
    const int total = nplanes * data_words;
    const FastDiv div_dw((uint32_t)max(data_words, 1)), div_nc((uint32_t)nc);
    const int64_t img_stride = (int64_t)a.C * a.H * a.W;
    const float* base = a.x + ((int64_t)n_lo * a.C + c_lo) * a.H * a.W + (int64_t)h_lo * a.W;
    for (int f0 = warp; f0 < total; f0 += 8 * 16) {
      float v[16];
#pragma unroll
      for (int u = 0; u < 16; ++u) {
        const int f = min(f0 + 8 * u, total - 1);
        const int pl = (int)div_dw.div((uint32_t)f), q = f - pl * data_words;
        const int nn = (int)div_nc.div((uint32_t)pl), c = pl - nn * nc;
        const int e = 32 * q + lane;
        v[u] = __ldg(base + nn * img_stride + (int64_t)c * a.H * a.W + min(e, plane_bits - 1));
        if (e >= plane_bits) v[u] = 0.0f;
      }
#pragma unroll
      for (int u = 0; u < 16; ++u) {
        const uint32_t word = __ballot_sync(0xFFFFFFFFu, v[u] > 0.0f);
        const int f = f0 + 8 * u;
        if (lane == 0 && f < total) {
          const int pl = (int)div_dw.div((uint32_t)f);
          stream[pl * plane_words + a.guard + (f - pl * data_words)] = word;
        }
      }
    }
  }
  for (int e = threadIdx.x; e < nplanes * 2 * a.guard; e += 256) {
    const int pl = e / (2 * a.guard), g = e - pl * 2 * a.guard;
    stream[pl * plane_words + (g < a.guard ? g : data_words + g)] = 0u;
  }
  __syncthreads();
  // 2. the 32 x 32 blocks of columns kb .. kb + 31
  const int kb = k0 + 32 * warp;
  // column k = kb + lane as (channel, kernel row, kernel column), fixed for the whole tile
  const int kl = min(kb + lane, a.K - 1);
  const int cl_ = (int)a.div_khw.div((uint32_t)kl), tl_ = kl - cl_ * a.khw;
  const int il_ = (int)a.div_kw.div((uint32_t)tl_), jl_ = tl_ - il_ * a.kw;
  const int Ho = a.HWo / a.Wo;
  for (int sub = 0; sub < nsub; ++sub) {
    const int ms = m0 + 32 * sub;
    uint32_t roww = 0, colw = 0;
    if (kb < a.K && ms < a.M) {  // warp-uniform
      if (a.same) {
        // "same" convolution: pixel p of an image reads input position p + (i - pad) W + (j - pad)
        // for tap (i, j), so the column word of k over 32 pixels of one image is one 32-bit window
        // of the plane stream (rows outside the image fall in the zero guards), masked where
        // the tap's input column leaves the image row
        const int n = (int)a.div_hwo.div((uint32_t)ms), p0 = ms - n * a.HWo;
        if (kb + lane < a.K) {
          const int lo = max(0, a.pad - jl_), hi = min(a.W, a.W + a.pad - jl_);  // valid output columns
          uint32_t mask;
          if (32 % a.W == 0) {
            const uint32_t row = (a.W == 32 ? 0xFFFFFFFFu : ((1u << hi) - (1u << lo)));
            mask = a.W == 32 ? (hi >= 32 ? 0xFFFFFFFFu << lo : ((1u << hi) - 1u) & (0xFFFFFFFFu << lo))
                             : row * (0xFFFFFFFFu / ((1u << a.W) - 1u));
          } else {
            mask = 0u;
            int t = p0 - (int)a.div_wo.div((uint32_t)p0) * a.Wo;  // output column of bit 0
            for (int b = 0; b < 32;) {
              const int seg = min(a.W - t, 32 - b);
              const int s0 = max(lo - t, 0), s1 = min(hi - t, seg);
              if (s1 > s0) mask |= ((s1 - s0 >= 32) ? 0xFFFFFFFFu : ((1u << (s1 - s0)) - 1u)) << (b + s0);
              b += seg;
              t = 0;
            }
          }
          const uint32_t* st = stream + ((n - n_lo) * nc + (cl_ - c_lo)) * plane_words;
          const int pos = gbits + p0 - h_lo * a.W + (il_ - a.pad) * a.W + (jl_ - a.pad);
          colw = stream_bits(st, pos, 32) & mask;
        }
        roww = warp_transpose32(colw, lane);
      } else if (a.stride == 1) {
        // column word of k = kb + lane over pixels ms .. ms + 31: runs along output rows
        const int mend = min(a.M, ms + 32);
        int n = (int)a.div_hwo.div((uint32_t)ms), rem = ms - n * a.HWo;
        int oh = (int)a.div_wo.div((uint32_t)rem), ow = rem - oh * a.Wo;
        const uint32_t* st_c = stream + (cl_ - c_lo) * plane_words;
        const bool kvalid = kb + lane < a.K;
        for (int m = ms; m < mend;) {
          const int cnt = min(a.Wo - ow, mend - m);  // pixels left on this output row
          const int h = oh - a.pad + il_;
          const int wa = ow - a.pad + jl_;  // input column of the run's first pixel
          const int lo = max(0, -wa), hi = min(cnt, a.W - wa);
          if (kvalid && h >= 0 && h < a.H && hi > lo) {
            const uint32_t* st = st_c + (n - n_lo) * nc * plane_words;
            colw |= stream_bits(st, gbits + (h - h_lo) * a.W + wa + lo, hi - lo) << (m - ms + lo);
          }
          m += cnt;
          ow += cnt;
          if (ow == a.Wo) {
            ow = 0;
            if (++oh == Ho) { oh = 0; ++n; }
          }
        }
        roww = warp_transpose32(colw, lane);
      } else if (a.stride == 2) {
        // stride 2: the column word of k = kb + lane over pixels ms .. ms + 31, by runs along
        // output rows as for stride 1; a run of pixels ow .. ow + cnt - 1 reads every other bit
        // of its input row from input column 2 ow - pad + j, so its bits are the even bits of a
        // stream window of at most 63 bits (stream_even_bits)
        const int mend = min(a.M, ms + 32);
        int n = (int)a.div_hwo.div((uint32_t)ms), rem = ms - n * a.HWo;
        int oh = (int)a.div_wo.div((uint32_t)rem), ow = rem - oh * a.Wo;
        const uint32_t* st_c = stream + (cl_ - c_lo) * plane_words;
        const bool kvalid = kb + lane < a.K;
        for (int m = ms; m < mend;) {
          const int cnt = min(a.Wo - ow, mend - m);  // pixels left on this output row
          const int h = 2 * oh - a.pad + il_;
          const int wa = 2 * ow - a.pad + jl_;  // input column of the run's first pixel
          // pixels t of the run whose input column wa + 2 t lies in [0, W)
          const int lo = wa >= 0 ? 0 : (1 - wa) / 2;
          const int hi = wa <= a.W - 1 ? min(cnt, (a.W - 1 - wa) / 2 + 1) : 0;
          if (kvalid && h >= 0 && h < a.H && hi > lo) {
            const uint32_t* st = st_c + (n - n_lo) * nc * plane_words;
            colw |= stream_even_bits(st, gbits + (h - h_lo) * a.W + wa + 2 * lo, hi - lo) << (m - ms + lo);
          }
          m += cnt;
          ow += cnt;
          if (ow == a.Wo) {
            ow = 0;
            if (++oh == Ho) { oh = 0; ++n; }
          }
        }
        roww = warp_transpose32(colw, lane);
      } else {
        // row word of pixel ms + lane over columns kb .. kb + 31: runs along kernel rows
        const int mr = ms + lane;
        if (mr < a.M) {
          const int n = (int)a.div_hwo.div((uint32_t)mr), rem = mr - n * a.HWo;
          const int oh = (int)a.div_wo.div((uint32_t)rem), ow = rem - oh * a.Wo;
          const int h0 = oh * a.stride - a.pad, w0 = ow * a.stride - a.pad;
          int c = (int)a.div_khw.div((uint32_t)kb), t = kb - c * a.khw;
          int i = (int)a.div_kw.div((uint32_t)t), j = t - i * a.kw;
          const int kend = min(a.K, kb + 32);
          const uint32_t* st_n = stream + (n - n_lo) * nc * plane_words;
          for (int k = kb; k < kend;) {
            const int cnt = min(a.kw - j, kend - k);  // taps left on this kernel row
            const int h = h0 + i;
            const int wa = w0 + j;
            const int lo = max(0, -wa), hi = min(cnt, a.W - wa);
            if (h >= 0 && h < a.H && hi > lo)
              roww |= stream_bits(st_n + (c - c_lo) * plane_words, gbits + (h - h_lo) * a.W + wa + lo, hi - lo)
                      << (k - kb + lo);
            k += cnt;
            j += cnt;
            if (j == a.kw) {
              j = 0;
              if (++i == a.kh) { i = 0; ++c; }
            }
          }
        }
        colw = warp_transpose32(roww, lane);
      }
    }
    rw_s[32 * sub + lane][warp] = roww;
    cw_s[32 * warp + lane][sub] = colw;
  }
  __syncthreads();
  // 3. outputs
  if (a.row_bits) {
    const int64_t w0 = (int64_t)blockIdx.x * 8;
    for (int e = threadIdx.x; e < (m1 - m0) * 8; e += 256) {
      const int r = e >> 3, q = e & 7;
      if (w0 + q < a.row_words) a.row_bits[(int64_t)(m0 + r) * a.row_words + w0 + q] = rw_s[r][q];
    }
  }
  if (have_k && (a.col_bits || a.colsum)) {
    const int64_t wbase = m0 / 32;
    if (a.col_bits) {
      for (int e = threadIdx.x; e < (k1 - k0) * nsub; e += 256) {
        const int kk = e / nsub, sub = e - kk * nsub;
        if (wbase + sub < a.col_words) a.col_bits[(int64_t)(k0 + kk) * a.col_words + wbase + sub] = cw_s[kk][sub];
      }
    }
    if (a.colsum) {
      for (int kk = threadIdx.x; kk < k1 - k0; kk += 256) {
        int sum = 0;
        for (int sub = 0; sub < nsub; ++sub) {
          const int valid = min(32, max(0, a.M - (m0 + 32 * sub)));
          sum += 2 * __popc(cw_s[kk][sub]) - valid;
        }
        atomicAdd(a.colsum + k0 + kk, sum);
      }
    }
  }
}

// ---------------------------------------------------------------------------
// Unfolder for "same" convolutions (stride 1, kh = kw = 2 pad + 1, so Ho = H and Wo = W)
// whose planes hold a multiple of 32 pixels and whose tiles hold whole images: a tile is
// 32 NSUB pixels = ipt images x 256 columns.
//  1. The input region of a tile (ipt images x nc channels, whole planes) is, per image,
//     one contiguous run of x, so sign-packing it is a linear copy into shared memory:
//     word f of the region is the ballot of 32 consecutive floats.  Planes lie back to back
//     (dw = H W / 32 words each); zero guard words sit only before and after the region.
//  2. Pixel p reads input pixel p + (i - pad) W + (j - pad) for tap (i, j), so the column
//     word of k over 32 pixels of one image is a 32-bit window of its channel's plane.  It
//     is masked to the pixels whose tap lands inside the image: a pixel interval for the
//     input row (reads that cross into a neighbouring plane fall outside it) and a per-j
//     pattern for the input column.  The shuffle transpose gives the row words.
//  3. Row words and column words go through XOR-swizzled shared memory (conflict-free
//     32-lane writes) and leave as 16-byte stores; the column sums come from the same reads.
struct UnfoldSameArgs {
  const float* x;
  const uint32_t* planes;  // or the sign bits of x as planes [N][C][dw] words (then x is unused)
  uint32_t* row_bits;
  uint32_t* col_bits;
  int32_t* colsum;
  int64_t row_words, col_words;
  int N, C, H, W, pad, kw, khw, K, HW;
  int dw;        // words per plane, H W / 32
  int ipt;       // images per tile, 32 NSUB / (H W)
  int guard;     // zero words before and after the region
  uint32_t rep;  // W divides 32: replicates a W-bit row pattern over 32 bits (1 for W = 32); else 0
  FastDiv div_khw, div_kw;
  // optional e4m3 copies of the signs (+1 = 0x38, -1 = 0xB8): rows [M][ld_row_e] (row r = pixel,
  // byte k) and columns [K][ld_col_e] (row k, byte r); the bytes from the valid length to the
  // next multiple of 16 are written as 0
  uint8_t* row_e4m3;
  uint8_t* col_e4m3;
  int64_t ld_row_e, ld_col_e, M;
};

// 16 signs (bits 0..15 of w) as 16 e4m3 bytes, the bytes at or past `valid` zero.
__device__ __forceinline__ uint4 e4m3_signs16(uint32_t w, int valid) {
  uint4 v = make_uint4(e4m3_signs4(w & 15u), e4m3_signs4((w >> 4) & 15u), e4m3_signs4((w >> 8) & 15u),
                       e4m3_signs4((w >> 12) & 15u));
  if (valid < 16) {
    uint32_t* p = &v.x;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int keep = min(max(valid - 4 * q, 0), 4);  // bytes of word q that stay
      p[q] &= keep == 4 ? 0xFFFFFFFFu : ((1u << (8 * keep)) - 1u);
    }
  }
  return v;
}

__device__ __forceinline__ uint32_t bit_range(int lo, int hi) {  // bits lo .. hi - 1 of a word
  lo = max(lo, 0);
  hi = min(hi, 32);
  if (hi <= lo) return 0u;
  return (hi - lo == 32 ? 0xFFFFFFFFu : ((1u << (hi - lo)) - 1u)) << lo;
}

// 4 words read as one 16-byte vector from a chunk whose words were stored at index ^ z
// (z in 0..3): word e of the result is the vector's word e ^ z.
__device__ __forceinline__ uint4 unswizzle4(uint4 v, int z) {
  if (z & 2) v = make_uint4(v.z, v.w, v.x, v.y);
  if (z & 1) v = make_uint4(v.y, v.x, v.w, v.z);
  return v;
}

template <int NSUB>
__global__ void __launch_bounds__(256) unfold_same_kernel(UnfoldSameArgs a) {
  static_assert(NSUB == 4 || NSUB == 8, "tiles of 128 or 256 pixels");
  constexpr int TM = 32 * NSUB;
  constexpr int kZShift = NSUB == 4 ? 3 : 2;  // column-word swizzle: (k >> kZShift) & (NSUB - 1)
  FQT1_PDL_WAIT();
  FQT1_PDL_TRIGGER();
  extern __shared__ uint32_t region[];
  __shared__ __align__(16) uint32_t rw_s[TM * 8];     // [pixel][8 k-words], word q at q ^ ((pixel >> 2) & 7)
  __shared__ __align__(16) uint32_t cw_s[256 * NSUB];  // [k][NSUB pixel-words], word s at s ^ z(k)
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_lo = blockIdx.y * a.ipt;
  const int nimg = min(a.ipt, a.N - n_lo);
  const int k0 = blockIdx.x * 256, k1 = min(a.K, k0 + 256);
  const int c_lo = (int)a.div_khw.div((uint32_t)k0);
  const int nc = (int)a.div_khw.div((uint32_t)(k1 - 1)) - c_lo + 1;
  const int span = nc * a.dw;  // region words per image
  const int total = nimg * span;
  uint32_t* st = region + a.guard;
  // 1. sign-pack; f / span by a multiply-high with ceil(2^32 / span) (exact for f, span < 2^16)
  {
    const uint32_t inv = (uint32_t)(0xFFFFFFFFu / (uint32_t)span) + 1u;
    const float* src = a.x + ((int64_t)n_lo * a.C + c_lo) * a.HW + lane;
    const int64_t img_stride = (int64_t)a.C * a.HW;
    if (a.planes) {  // the signs given as plane bits: the region is a copy of plane words
      const uint32_t* ps = a.planes + ((int64_t)n_lo * a.C + c_lo) * a.dw;
      const int64_t img_w = (int64_t)a.C * a.dw;
      for (int f = threadIdx.x; f < total; f += 256) {
        const int img = (int)__umulhi((uint32_t)f, inv);
        st[f] = __ldg(ps + img * img_w + (f - img * span));
      }
    }
    for (int f0 = warp; !a.planes && f0 < total; f0 += 8 * 16) {
      // unconditional loads from clamped word indices (the ballots of words past the region are
      // not stored): a load under a condition is not hoisted, and the 16 round trips serialize
      float v[16];
#pragma unroll
      for (int u = 0; u < 16; ++u) {
        const int f = min(f0 + 8 * u, total - 1);
        const int img = (int)__umulhi((uint32_t)f, inv);
        v[u] = __ldg(src + img * img_stride + (int64_t)(f - img * span) * 32);
      }
#pragma unroll
      for (int u = 0; u < 16; ++u) {
        const uint32_t word = __ballot_sync(0xFFFFFFFFu, v[u] > 0.0f);
        if (lane == 0 && f0 + 8 * u < total) st[f0 + 8 * u] = word;
      }
    }
    for (int e = threadIdx.x; e < 2 * a.guard; e += 256) region[e < a.guard ? e : total + e] = 0u;
  }
  __syncthreads();
  // 2. column word of k = kb + lane over each 32-pixel sub-tile, and its transpose
  const int kb = k0 + 32 * warp;
  const int k = kb + lane;
  const bool kvalid = k < k1;
  const int kk = min(k, a.K - 1);
  const int c = (int)a.div_khw.div((uint32_t)kk), t = kk - c * a.khw;
  const int i = (int)a.div_kw.div((uint32_t)t), j = t - i * a.kw;
  const int plo = max(0, a.pad - i) * a.W, phi = min(a.H, a.H + a.pad - i) * a.W;  // pixels with the row inside
  const int olo = max(0, a.pad - j), ohi = min(a.W, a.W + a.pad - j);              // output columns inside
  const uint32_t cmask_rep = a.rep ? bit_range(olo, ohi) * a.rep : 0u;
  // bit position, relative to st, of the window of pixel 0 of image 0
  const int pos0 = 32 * (c - c_lo) * a.dw + (i - a.pad) * a.W + (j - a.pad);
  int img = 0, q = 0, ow0 = 0;  // sub-tile s = img dw + q; ow0 = output column of its bit 0
#pragma unroll 1
  for (int s = 0; s < NSUB; ++s) {
    uint32_t colw = 0;
    if (kvalid && img < nimg) {
      const int p0 = 32 * q;
      const int pos = pos0 + 32 * img * span + p0;
      const int w = pos >> 5, o = pos & 31;
      const uint64_t v = ((uint64_t)st[w + 1] << 32) | st[w];
      uint32_t cmask = cmask_rep;
      if (!a.rep) {
        for (int b = 0, tt = ow0; b < 32;) {
          const int seg = min(a.W - tt, 32 - b);
          cmask |= bit_range(b + max(olo - tt, 0), b + min(ohi - tt, seg));
          b += seg;
          tt = 0;
        }
      }
      colw = (uint32_t)(v >> o) & bit_range(plo - p0, phi - p0) & cmask;
    }
    if (a.row_bits || a.row_e4m3) {  // uniform: a caller that needs only the column packing skips the transposes
      const uint32_t roww = warp_transpose32(colw, lane);
      const int px = 32 * s + lane;
      rw_s[px * 8 + (warp ^ ((px >> 2) & 7))] = roww;
    }
    const int kl = 32 * warp + lane;
    cw_s[kl * NSUB + (s ^ ((kl >> kZShift) & (NSUB - 1)))] = colw;
    if (!a.rep) {
      ow0 += 32;
      while (ow0 >= a.W) ow0 -= a.W;
    }
    if (++q == a.dw) { q = 0; ++img; ow0 = 0; }
  }
  __syncthreads();
  // 3. outputs as 16-byte chunks
  if (a.row_bits) {
    const int64_t wbase = (int64_t)k0 / 32;
    for (int e = threadIdx.x; e < 2 * TM; e += 256) {
      const int px = e >> 1, h = e & 1;
      const int sw = (px >> 2) & 7;
      if (px < nimg * a.HW && wbase + 4 * h < a.row_words) {
        const uint4 v = unswizzle4(*reinterpret_cast<const uint4*>(rw_s + px * 8 + 4 * (h ^ (sw >> 2))), sw & 3);
        *reinterpret_cast<uint4*>(a.row_bits + ((int64_t)n_lo * a.HW + px) * a.row_words + wbase + 4 * h) = v;
      }
    }
  }
  if (a.row_e4m3) {  // 16 bytes per chunk, 16 chunks (256 columns) per pixel
    for (int e = threadIdx.x; e < 16 * TM; e += 256) {
      const int px = e >> 4, ch = e & 15;
      const int64_t kc = (int64_t)k0 + 16 * ch;
      if (px < nimg * a.HW && kc < a.K) {
        const int sw = (px >> 2) & 7;
        const uint32_t word = rw_s[px * 8 + ((ch >> 1) ^ sw)] >> (16 * (ch & 1));
        const uint4 v = e4m3_signs16(word, (int)(a.K - kc < 16 ? a.K - kc : 16));
        *reinterpret_cast<uint4*>(a.row_e4m3 + ((int64_t)n_lo * a.HW + px) * a.ld_row_e + kc) = v;
      }
    }
  }
  if (a.col_e4m3) {  // TM bytes per column k: a warp writes four columns' contiguous runs
    constexpr int kChunks = TM / 16;
    const int64_t p0 = (int64_t)blockIdx.y * TM;
    for (int e = threadIdx.x; e < 256 * kChunks; e += 256) {
      const int kl = e / kChunks, ch = e % kChunks;
      const int64_t pc = p0 + 16 * ch;
      if (k0 + kl < k1 && pc < a.M) {
        const int z = (kl >> kZShift) & (NSUB - 1);
        const int wi = ch >> 1;  // pixel word of the chunk
        const uint32_t word = cw_s[kl * NSUB + (wi ^ z)] >> (16 * (ch & 1));
        const uint4 v = e4m3_signs16(word, (int)(a.M - pc < 16 ? a.M - pc : 16));
        *reinterpret_cast<uint4*>(a.col_e4m3 + (int64_t)(k0 + kl) * a.ld_col_e + pc) = v;
      }
    }
  }
  {
    const int kl = threadIdx.x;
    if (k0 + kl < k1) {
      const int z = (kl >> kZShift) & (NSUB - 1);
      const int64_t wbase = (int64_t)blockIdx.y * NSUB;
      int ones = 0;
#pragma unroll
      for (int h = 0; h < NSUB / 4; ++h) {
        const uint4 v = unswizzle4(*reinterpret_cast<const uint4*>(cw_s + kl * NSUB + 4 * (h ^ (z >> 2))), z & 3);
        ones += __popc(v.x) + __popc(v.y) + __popc(v.z) + __popc(v.w);
        if (a.col_bits && wbase + 4 * h < a.col_words)
          *reinterpret_cast<uint4*>(a.col_bits + (int64_t)(k0 + kl) * a.col_words + wbase + 4 * h) = v;
      }
      if (a.colsum) atomicAdd(a.colsum + k0 + kl, 2 * ones - nimg * a.HW);
    }
  }
}

template <class Loader>
static fqt1_status launch_pack(const Loader& L, uint32_t* row_bits, uint32_t* col_bits, int32_t* colsum,
                               cudaStream_t s) {
  const int64_t row_words = fqt1_packed_words(L.cols);
  const int64_t col_words = fqt1_packed_words(L.rows);
  const int64_t row_tiles = (L.rows + Loader::kRows - 1) / Loader::kRows;
  const int64_t word_tiles = (row_words + kPackWordsPerCta - 1) / kPackWordsPerCta;
  const int64_t col_words_written = (L.rows + 31) / 32;
  if (row_tiles > 65535) return FQT1_ERR_UNSUPPORTED;
  if (colsum) FQT1_CUDA_TRY(cudaMemsetAsync(colsum, 0, sizeof(int32_t) * L.cols, s));
  dim3 grid((unsigned)word_tiles, (unsigned)row_tiles);
  launch_k(pack_kernel<Loader>, dim3(grid), dim3(256), 0, s, L, row_bits, row_words, col_bits, col_words, colsum);
  fqt1_count_launches(1);
  FQT1_CUDA_TRY(cudaGetLastError());
  if (col_bits && col_words > col_words_written) {
    const int64_t n = L.cols * (col_words - col_words_written);
    launch_k(zero_col_pad_kernel, dim3((unsigned)((n + 255) / 256)), dim3(256), 0, s, col_bits, L.cols, col_words,
                                                                    col_words_written);
    fqt1_count_launches(1);
    FQT1_CUDA_TRY(cudaGetLastError());
  }
  return FQT1_OK;
}


// ------------------------------------------------------------------ implicit-convolution packings
// Pixel-major signs of x [N, C, H, W] for the implicit-GEMM forward: word b of pixel
// p = (n H + h) W + w holds sign(x[n, 32 b + e, h, w]) > 0 at bit e.  A CTA takes 32
// consecutive pixels (lane = pixel) and 4 blocks of 32 channels (warp = block): 32 loads
// per lane, each a contiguous run of the plane across the warp, then one word per lane; the
// 4 words of a pixel leave as one 16-byte store.
constexpr int kPixBlocks = 4;
__global__ void __launch_bounds__(32 * kPixBlocks) pack_pixels_kernel(const float* __restrict__ x, int64_t P, int C,
                                                                      int HW, FastDiv div_hw, int64_t words,
                                                                      uint32_t* __restrict__ out) {
  FQT1_PDL_WAIT();
  FQT1_PDL_TRIGGER();
  __shared__ __align__(16) uint32_t w_s[32][kPixBlocks];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t p = (int64_t)blockIdx.x * 32 + lane;
  const uint32_t pc = (uint32_t)min(p, P - 1);
  const uint32_t n = div_hw.div(pc);
  const int cb = blockIdx.y * kPixBlocks + warp;  // C is a multiple of 32 kPixBlocks
  const float* src = x + ((int64_t)n * C + 32 * cb) * HW + (pc - n * (uint32_t)HW);
  float v[32];
#pragma unroll
  for (int u = 0; u < 32; ++u) v[u] = __ldg(src + (int64_t)u * HW);
  uint32_t wd = 0;
#pragma unroll
  for (int u = 0; u < 32; ++u) wd |= (v[u] > 0.0f ? 1u : 0u) << u;
  w_s[lane][warp] = wd;
  __syncthreads();
  const int64_t q = (int64_t)blockIdx.x * 32 + threadIdx.x;  // one pixel per thread of warp 0
  if (threadIdx.x < 32 && q < P)
    *reinterpret_cast<uint4*>(out + q * words + (int64_t)blockIdx.y * kPixBlocks) =
        *reinterpret_cast<const uint4*>(&w_s[threadIdx.x][0]);
}

// Tap-major signs of w [D, C, kh, kw] for the implicit-GEMM forward: row d, contraction index
// k' = t C + c for tap t = i kw + j, i.e. word t C / 32 + b holds sign(w[d, 32 b + e, i, j]) at
// bit e.  One warp per (d, t); lane = channel within a block of 32, one ballot per block (8
// loads in flight per lane), lane b keeps word b of its group of 32 blocks.  Words past
// kh kw C / 32 (the row padding to 16 bytes) are written as 0.
__global__ void __launch_bounds__(256) pack_weight_taps_kernel(const float* __restrict__ w, int64_t D, int C, int khw,
                                                               int64_t words, uint32_t* __restrict__ out) {
  FQT1_PDL_WAIT();
  FQT1_PDL_TRIGGER();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t g = (int64_t)blockIdx.x * 8 + warp;
  const int64_t d = g / khw;
  const int t = (int)(g - d * khw);
  if (d >= D) return;  // warp-uniform
  const float* src = w + d * (int64_t)C * khw + t;
  uint32_t* dst = out + d * words + (int64_t)t * (C / 32);
  const int nb = C / 32;
  for (int b0 = 0; b0 < nb; b0 += 32) {
    uint32_t mine = 0;
    for (int b1 = b0; b1 < min(nb, b0 + 32); b1 += 8) {
      float v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) v[u] = __ldg(src + (int64_t)(min(b1 + u, nb - 1) * 32 + lane) * khw);
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const uint32_t wd = __ballot_sync(0xFFFFFFFFu, v[u] > 0.0f);
        if (lane == b1 + u - b0) mine = wd;
      }
    }
    if (b0 + lane < nb) dst[b0 + lane] = mine;
  }
  if (t == khw - 1) {
    const int64_t used = (int64_t)khw * nb;
    for (int64_t e = used + lane; e < words; e += 32) out[d * words + e] = 0u;
  }
}

// ------------------------------------------------------------------ e4m3 signs
// e4m3 bytes of packed signs (the B operand of the products when it is loaded as bytes):
// out[r][e] = 0x38 (+1) where bit e of row r is set, 0xB8 (-1) where it is clear, for e < n,
// and 0 for n <= e < ld_out (so that no byte past the contraction is a NaN pattern).  One thread
// per 16 output bytes; bit k of a nibble lands on the sign bit of byte k through one multiply.
__global__ void __launch_bounds__(256) expand_signs_kernel(const uint32_t* __restrict__ bits, int64_t rows, int64_t n,
                                                           int64_t ld_words, uint8_t* __restrict__ out, int64_t ld_out) {
  FQT1_PDL_WAIT();
  FQT1_PDL_TRIGGER();
  const int64_t chunks = ld_out / 16;
  const int64_t t = (int64_t)blockIdx.x * 256 + threadIdx.x;
  if (t >= rows * chunks) return;
  const int64_t r = t / chunks, e0 = 16 * (t - r * chunks);
  const uint32_t h = e0 < n ? (__ldg(bits + r * ld_words + (e0 >> 5)) >> (e0 & 16)) & 0xFFFFu : 0u;
  uint32_t wv[4];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    uint32_t v = (((h >> (4 * q)) & 15u) * 0x10204080u & 0x80808080u) ^ 0xB8B8B8B8u;
#pragma unroll
    for (int b = 0; b < 4; ++b)
      if (e0 + 4 * q + b >= n) v &= ~(0xFFu << (8 * b));
    wv[q] = v;
  }
  *reinterpret_cast<uint4*>(out + r * ld_out + e0) = make_uint4(wv[0], wv[1], wv[2], wv[3]);
}

// ------------------------------------------------------------------ channels-last input
// Sign bits of a channels-last x (N, H, W, C in memory) as planes [N][C][pw], pw = ceil(H W / 32):
// bit e of word q of plane (n, c) is sign(x[n, c, pixel 32 q + e]) > 0.  A warp takes 32 pixels x
// 32 channels: lane p reads its pixel's 32 channels (128 contiguous bytes), forms their sign
// word, and the warp transpose turns the 32 pixel words into the 32 plane words.
__global__ void __launch_bounds__(256) pack_planes_nhwc_kernel(const float* __restrict__ x, int N, int C, int HW,
                                                               int pw, uint32_t* __restrict__ planes) {
  FQT1_PDL_WAIT();
  FQT1_PDL_TRIGGER();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int cbs = C / 32;
  const int64_t units = (int64_t)N * pw * cbs;
  for (int64_t u = (int64_t)blockIdx.x * 8 + warp; u < units; u += (int64_t)gridDim.x * 8) {  // warp-uniform
    const int64_t n = u / ((int64_t)pw * cbs);
    const int rem = (int)(u - n * pw * cbs), q = rem / cbs, cb = rem - q * cbs;
    const int p = 32 * q + lane;
    const float4* src = reinterpret_cast<const float4*>(x + ((n * HW + min(p, HW - 1)) * C + 32 * cb));
    float4 v[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) v[k] = __ldg(src + k);
    uint32_t wd = 0;
#pragma unroll
    for (int k = 0; k < 8; ++k)
      wd |= (v[k].x > 0.f ? 1u : 0u) << (4 * k) | (v[k].y > 0.f ? 2u : 0u) << (4 * k) |
            (v[k].z > 0.f ? 4u : 0u) << (4 * k) | (v[k].w > 0.f ? 8u : 0u) << (4 * k);
    if (p >= HW) wd = 0u;
    const uint32_t pwd = warp_transpose32(wd, lane);  // lane c: channel 32 cb + c over the 32 pixels
    planes[(n * C + 32 * cb + lane) * pw + q] = pwd;
  }
}
// Sign bits of a contiguous [N, C, H, W] x as channel planes [N C][pw] words, pw = ceil(H W / 32):
// bit e of word q of plane p is x[p H W + 32 q + e] > 0, bits past H W clear.  A warp takes 8
// consecutive words of one plane and has its 8 coalesced 128-byte loads in flight together; a
// word is the ballot of its 32 floats.
__global__ void __launch_bounds__(256) pack_planes_nchw_kernel(const float* __restrict__ x, int64_t planes_n, int HW,
                                                               int pw, uint32_t* __restrict__ planes) {
  FQT1_PDL_WAIT();
  FQT1_PDL_TRIGGER();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int blocks = (pw + 7) / 8;
  const int64_t units = planes_n * blocks;
  for (int64_t u = (int64_t)blockIdx.x * 8 + warp; u < units; u += (int64_t)gridDim.x * 8) {  // warp-uniform
    const int64_t pl = u / blocks;
    const int q0 = 8 * (int)(u - pl * blocks);
    const float* src = x + pl * HW;
    float v[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) v[k] = __ldg(src + min(32 * (q0 + k) + lane, HW - 1));
    uint32_t mine = 0u;
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const uint32_t wd = __ballot_sync(0xFFFFFFFFu, v[k] > 0.0f && 32 * (q0 + k) + lane < HW);
      if (lane == k) mine = wd;
    }
    if (lane < 8 && q0 + lane < pw) planes[pl * pw + q0 + lane] = mine;
  }
}
// Unfolder of a pointwise convolution (1 x 1 window, no padding, any stride): X_u[m][c] is
// sign(x[n][c][s oh][s ow]), a strided subsample of x.  A warp takes 32 output pixels x 32
// channels (lane = channel): its 32 loads per lane (one per pixel) are in flight together, a
// ballot per pixel gives that pixel's row word, and each lane's own 32 compares give its
// channel's column word.  Pixel groups run up to the padded column words and channel groups up
// to the padded row words, so the padding words are written as zeros.  The column sums are
// reduced over the CTA's 8 warps (same channels) before one atomic per channel.
struct UnfoldPointArgs {
  const float* x;
  uint32_t* row_bits;
  uint32_t* col_bits;
  int32_t* colsum;
  int64_t row_words, col_words;
  int C, H, W, stride, Ho, Wo, M;
  FastDiv div_hwo, div_wo;
};

__global__ void __launch_bounds__(256) unfold_pointwise_kernel(UnfoldPointArgs a) {
  FQT1_PDL_WAIT();
  FQT1_PDL_TRIGGER();
  __shared__ int32_t cs_s[8][32];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t pg = (int64_t)blockIdx.x * 8 + warp;  // pixel group (32 pixels)
  const int cw = blockIdx.y;                           // channel word
  const int c = cw * 32 + lane;
  const bool cvalid = c < a.C;
  const int64_t m0 = pg * 32;
  int32_t cnt = 0;
  if (pg < a.col_words) {  // warp-uniform
    // input offset of pixel m0 (clamped) for channel c; later pixels step along the output row
    const int mc = (int)(m0 < a.M - 1 ? m0 : a.M - 1);
    int n = (int)a.div_hwo.div((uint32_t)mc), rem = mc - n * a.Ho * a.Wo;
    int oh = (int)a.div_wo.div((uint32_t)rem), ow = rem - oh * a.Wo;
    const int64_t plane = (int64_t)a.H * a.W, cc = cvalid ? c : a.C - 1;
    float v[32];
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      v[j] = __ldg(a.x + ((int64_t)n * a.C + cc) * plane + (int64_t)oh * a.stride * a.W + (int64_t)ow * a.stride);
      if (m0 + j + 1 < a.M) {  // the next pixel (uniform); past M the last one is loaded again
        if (++ow == a.Wo) { ow = 0; if (++oh == a.Ho) { oh = 0; ++n; } }
      }
    }
    uint32_t roww = 0u, colw = 0u;
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      const bool pvalid = m0 + j < a.M;
      const bool pos = v[j] > 0.0f && pvalid;
      const uint32_t b = __ballot_sync(0xFFFFFFFFu, pos && cvalid);
      if (lane == j) roww = b;
      colw |= (pos ? 1u : 0u) << j;
    }
    if (a.row_bits && m0 + lane < a.M && cw < a.row_words) a.row_bits[(m0 + lane) * a.row_words + cw] = roww;
    if (a.col_bits && cvalid) a.col_bits[(int64_t)c * a.col_words + pg] = colw;
    const int64_t left = a.M - m0;
    const int valid = left <= 0 ? 0 : (left >= 32 ? 32 : (int)left);
    cnt = cvalid ? 2 * __popc(colw) - valid : 0;
  }
  cs_s[warp][lane] = cnt;
  __syncthreads();
  if (a.colsum && warp == 0) {
    int32_t sum = 0;
#pragma unroll
    for (int w = 0; w < 8; ++w) sum += cs_s[w][lane];
    if (cvalid && sum != 0) atomicAdd(a.colsum + c, sum);
  }
}

// Planes of fewer than 32 pixels that divide 32 (4 x 4, 2 x 2, 1 x 1 maps): 32 consecutive floats
// of x are all the pixels of 32 / HW consecutive planes, so one ballot gives the words of all of
// them (one word per plane).  A warp takes 8 such chunks at a time, their loads in flight
// together.
__global__ void __launch_bounds__(256) pack_planes_small_kernel(const float* __restrict__ x, int64_t total, int HW,
                                                                uint32_t* __restrict__ planes) {
  FQT1_PDL_WAIT();
  FQT1_PDL_TRIGGER();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int per = 32 / HW;  // planes per chunk
  const uint32_t mask = (1u << HW) - 1u;
  const int64_t chunks = (total + 31) / 32;
  for (int64_t c0 = ((int64_t)blockIdx.x * 8 + warp) * 8; c0 < chunks; c0 += (int64_t)gridDim.x * 64) {
    float v[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) v[k] = __ldg(x + min((c0 + k) * 32 + lane, total - 1));
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      if (c0 + k >= chunks) break;  // warp-uniform
      const int64_t f = (c0 + k) * 32 + lane;
      const uint32_t wd = __ballot_sync(0xFFFFFFFFu, v[k] > 0.0f && f < total);
      const int64_t pl = (c0 + k) * per + lane;
      if (lane < per && pl * HW < total) planes[pl] = (wd >> (lane * HW)) & mask;
    }
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

extern "C" fqt1_status fqt1_binarize_pack(const float* x, int64_t rows, int64_t cols, int64_t ld,
                                          uint32_t* row_bits, uint32_t* col_bits, int32_t* colsum,
                                          void* stream) {
  if (!x || rows < 1 || cols < 1 || ld < cols) return FQT1_ERR_INVALID_ARG;
  if (!row_bits && !col_bits && !colsum) return FQT1_ERR_INVALID_ARG;
  if (!aligned16(x) || (row_bits && !aligned16(row_bits)) || (col_bits && !aligned16(col_bits)) ||
      (colsum && !aligned16(colsum)))
    return FQT1_ERR_MISALIGNED;
  cudaStream_t s = (cudaStream_t)stream;
  const int64_t row_words = fqt1_packed_words(cols), col_words = fqt1_packed_words(rows);
  const int64_t bands = (rows + 31) / 32;
  if (bands > 65535) return FQT1_ERR_UNSUPPORTED;
  if (colsum) FQT1_CUDA_TRY(cudaMemsetAsync(colsum, 0, sizeof(int32_t) * cols, s));
  if (cols % 4 == 0 && ld % 4 == 0)
    FQT1_CUDA_TRY(launch_k(pack_tile_kernel, dim3((unsigned)((cols + 32 * kPackTileWarps - 1) / (32 * kPackTileWarps)),
                                                  (unsigned)bands),
                           dim3(32 * kPackTileWarps), 0, s, x, rows, cols, ld, row_bits, row_words, col_bits, col_words,
                           colsum, (uint8_t*)nullptr, (int64_t)0, (uint8_t*)nullptr, (int64_t)0));
  else
    FQT1_CUDA_TRY(launch_k(pack_dense_kernel, dim3((unsigned)((row_words + 3) / 4), (unsigned)bands), dim3(128), 0,
                           s, x, rows, cols, ld, row_bits, row_words, col_bits, col_words, colsum));
  fqt1_count_launches(1);
  if (col_bits && col_words > bands) {
    const int64_t n = cols * (col_words - bands);
    FQT1_CUDA_TRY(launch_k(zero_col_pad_kernel, dim3((unsigned)((n + 255) / 256)), dim3(256), 0, s, col_bits, cols,
                           col_words, bands));
    fqt1_count_launches(1);
  }
  return FQT1_OK;
}

// Whether the whole-image Unfolder (unfold_same_kernel) serves the shape: a stride-1 "same"
// convolution whose tiles hold whole images (H W divides 128, or is 256), with its region and
// guards in 32 KB of shared memory.
static bool unfold_same_fits(int N, int C, int H, int W, int kh, int kw, int stride, int pad) {
  const int Ho = (H + 2 * pad - kh) / stride + 1, Wo = (W + 2 * pad - kw) / stride + 1;
  const int64_t Ki = (int64_t)C * kh * kw;
  const bool same = stride == 1 && kh == kw && kh == 2 * pad + 1 && (Ho * Wo) % 32 == 0;
  if (!(same && pad <= 32 && Ki < (1ll << 31) && (128 % (H * W) == 0 || H * W == 256))) return false;
  const int dw = H * W / 32, nsub = H * W == 256 ? 8 : 4, ipt = 32 * nsub / (H * W);
  const int guard = (pad * W + pad + 63) / 32;
  const int64_t nc_max = std::min<int64_t>(C, 256 / (kh * kw) + 2);
  const size_t smem = (size_t)(2 * guard + ipt * nc_max * dw) * 4;
  const int64_t row_tiles = (N + ipt - 1) / ipt;
  return row_tiles <= 65535 && smem <= 32 * 1024;
}

// A 1 x 1 window without padding: the pointwise Unfolder reads x directly.
static bool pointwise_conv(int kh, int kw, int pad) { return kh == 1 && kw == 1 && pad == 0; }

// Pixels per tile of the region Unfolder (unfold_bits_kernel): the largest of 256 (see below),
// 128, 64, 32 whose input region bound (images a tile may touch x channels of 256 columns x whole planes with
// guards) fits kUnfoldMaxStreamWords, with at most 65535 row tiles; 0 if none (gather path).
// Larger tiles pay the region set-up, its divisions and its barrier over more output words.
static int unfold_bits_tm(int N, int C, int H, int W, int kh, int kw, int stride, int pad) {
  const int Ho = (H + 2 * pad - kh) / stride + 1, Wo = (W + 2 * pad - kw) / stride + 1;
  const int64_t Mi = (int64_t)N * Ho * Wo, Ki = (int64_t)C * kh * kw;
  if (!(pad <= 32 && Ki < (1ll << 31))) return 0;
  const bool same = stride == 1 && kh == kw && kh == 2 * pad + 1 && (Ho * Wo) % 32 == 0;
  const int guard = same ? (pad * W + pad + 63) / 32 : 1;
  // 256-pixel tiles only for maps of 256 or more output pixels and windows larger than one tap
  // (measured: they speed up the stem, layer1 and the 32 x 32 layers, and slow down the 1 x 1
  // downsamples and the small maps)
  const int tm_max = (Ho * Wo >= 256 && kh * kw > 1) ? 256 : 128;
  for (int tm = tm_max; tm >= 32; tm /= 2) {
    const int64_t imgs = std::min<int64_t>(N, tm / (Ho * Wo) + 2);
    const int64_t chans = std::min<int64_t>(C, 256 / (kh * kw) + 2);
    const int64_t words = imgs * chans * (((int64_t)H * W + 31) / 32 + 2 * guard);
    if (words > kUnfoldMaxStreamWords) continue;
    return (Mi + tm - 1) / tm > 65535 ? 0 : tm;
  }
  return 0;
}

// The Unfolder of fqt1_im2col (x given) and of fqt1_im2col_planes (planes given: the sign bits of x
// as [N][C][ceil(H W / 32)] words; shapes that only the gather path serves are unsupported there).
static fqt1_status im2col_impl(const float* x, const uint32_t* planes, int32_t N, int32_t C, int32_t H, int32_t W,
                               int32_t kh, int32_t kw, int32_t stride, int32_t pad, uint32_t* row_bits,
                               uint32_t* col_bits, int32_t* colsum, void* stream, uint8_t* row_e4m3 = nullptr,
                               int64_t ld_re = 0, uint8_t* col_e4m3 = nullptr, int64_t ld_ce = 0) {
  if ((!x && !planes) || N < 1 || C < 1 || H < 1 || W < 1 || kh < 1 || kw < 1 || stride < 1 || pad < 0)
    return FQT1_ERR_INVALID_ARG;
  if (!row_bits && !col_bits && !colsum && !row_e4m3 && !col_e4m3) return FQT1_ERR_INVALID_ARG;
  const int64_t Ho64 = conv_extent(H, kh, stride, pad), Wo64 = conv_extent(W, kw, stride, pad);
  if (Ho64 == 0 || Wo64 == 0) return FQT1_ERR_INVALID_ARG;
  if (Ho64 < 0 || Wo64 < 0) return FQT1_ERR_UNSUPPORTED;
  const int Ho = (int)Ho64, Wo = (int)Wo64;
  if ((x && !aligned16(x)) || (row_bits && !aligned16(row_bits)) || (col_bits && !aligned16(col_bits)) ||
      (colsum && !aligned16(colsum)))
    return FQT1_ERR_MISALIGNED;
  if ((int64_t)N * C * H * W >= (1ll << 31) || (int64_t)N * Ho * Wo >= (1ll << 31)) return FQT1_ERR_UNSUPPORTED;
  cudaStream_t s = (cudaStream_t)stream;
  // Bit-level Unfolder when the input region of a tile fits in shared memory.  Bound on the
  // region of a tile of tm pixels: images it may touch x channels of 256 columns x whole planes.
  const int64_t Mi = (int64_t)N * Ho * Wo, Ki = (int64_t)C * kh * kw;
  const bool same = stride == 1 && kh == kw && kh == 2 * pad + 1 && (Ho * Wo) % 32 == 0;
  const bool e4m3 = row_e4m3 || col_e4m3;
  if (e4m3) {  // only the whole-image Unfolder writes the byte copies
    if (!unfold_same_fits(N, C, H, W, kh, kw, stride, pad)) return FQT1_ERR_UNSUPPORTED;
    if ((row_e4m3 && (ld_re < (Ki + 15) / 16 * 16 || ld_re % 16)) ||
        (col_e4m3 && (ld_ce < (Mi + 15) / 16 * 16 || ld_ce % 16)))
      return FQT1_ERR_INVALID_ARG;
    if ((row_e4m3 && !aligned16(row_e4m3)) || (col_e4m3 && !aligned16(col_e4m3))) return FQT1_ERR_MISALIGNED;
  }
  if (unfold_same_fits(N, C, H, W, kh, kw, stride, pad)) {
    // whole images per tile: the contiguous-region Unfolder
    UnfoldSameArgs u;
    u.x = x; u.planes = planes; u.row_bits = row_bits; u.col_bits = col_bits; u.colsum = colsum;
    u.row_e4m3 = row_e4m3; u.col_e4m3 = col_e4m3; u.ld_row_e = ld_re; u.ld_col_e = ld_ce; u.M = Mi;
    u.row_words = fqt1_packed_words(Ki); u.col_words = fqt1_packed_words(Mi);
    u.N = N; u.C = C; u.H = H; u.W = W; u.pad = pad; u.kw = kw; u.khw = kh * kw; u.K = (int)Ki; u.HW = H * W;
    u.dw = H * W / 32;
    const int nsub = H * W == 256 ? 8 : 4;
    u.ipt = 32 * nsub / (H * W);
    u.guard = (pad * W + pad + 63) / 32;
    u.rep = 32 % W == 0 ? (W == 32 ? 1u : 0xFFFFFFFFu / ((1u << W) - 1u)) : 0u;
    u.div_khw = FastDiv((uint32_t)(kh * kw)); u.div_kw = FastDiv((uint32_t)kw);
    const int64_t nc_max = std::min<int64_t>(C, 256 / (kh * kw) + 2);
    const size_t smem = (size_t)(2 * u.guard + u.ipt * nc_max * u.dw) * 4;
    const int64_t row_tiles = (N + u.ipt - 1) / u.ipt, word_tiles = (Ki + 255) / 256;
    if (row_tiles <= 65535 && smem <= 32 * 1024) {
      if (colsum) FQT1_CUDA_TRY(cudaMemsetAsync(colsum, 0, sizeof(int32_t) * Ki, s));
      if (nsub == 4)
        launch_k(unfold_same_kernel<4>, dim3((unsigned)word_tiles, (unsigned)row_tiles), dim3(256), smem, s, u);
      else
        launch_k(unfold_same_kernel<8>, dim3((unsigned)word_tiles, (unsigned)row_tiles), dim3(256), smem, s, u);
      fqt1_count_launches(1);
      FQT1_CUDA_TRY(cudaGetLastError());
      const int64_t written = row_tiles * nsub;
      if (col_bits && u.col_words > written) {
        const int64_t n = Ki * (u.col_words - written);
        launch_k(zero_col_pad_kernel, dim3((unsigned)((n + 255) / 256)), dim3(256), 0, s, col_bits, Ki, u.col_words,
                 written);
        fqt1_count_launches(1);
        FQT1_CUDA_TRY(cudaGetLastError());
      }
      return FQT1_OK;
    }
  }
  if (e4m3) return FQT1_ERR_UNSUPPORTED;
  if (x && pointwise_conv(kh, kw, pad) && Mi < (1ll << 31)) {
    // pointwise convolution: a strided subsample of x, read once per element
    UnfoldPointArgs u;
    u.x = x; u.row_bits = row_bits; u.col_bits = col_bits; u.colsum = colsum;
    u.row_words = fqt1_packed_words(Ki); u.col_words = fqt1_packed_words(Mi);
    u.C = C; u.H = H; u.W = W; u.stride = stride; u.Ho = Ho; u.Wo = Wo; u.M = (int)Mi;
    u.div_hwo = FastDiv((uint32_t)(Ho * Wo)); u.div_wo = FastDiv((uint32_t)Wo);
    if (colsum) FQT1_CUDA_TRY(cudaMemsetAsync(colsum, 0, sizeof(int32_t) * Ki, s));
    const int64_t gx = (u.col_words + 7) / 8;
    if (gx > 0x7FFFFFFF || u.row_words > 65535) return FQT1_ERR_UNSUPPORTED;
    launch_k(unfold_pointwise_kernel, dim3((unsigned)gx, (unsigned)u.row_words), dim3(256), 0, s, u);
    fqt1_count_launches(1);
    FQT1_CUDA_TRY(cudaGetLastError());
    return FQT1_OK;
  }
  if (const int tm = unfold_bits_tm(N, C, H, W, kh, kw, stride, pad)) {
    // 128-pixel tiles (smaller only when the input region does not fit): fewer CTAs, each
    // amortizing its region set-up over more output words
    // the fast path reads a 32-bit window up to pad W + pad bits before or after the plane
    const int guard = same ? (pad * W + pad + 63) / 32 : 1;
    {
      const int64_t imgs = std::min<int64_t>(N, tm / (Ho * Wo) + 2);
      const int64_t chans = std::min<int64_t>(C, 256 / (kh * kw) + 2);
      const int64_t words = imgs * chans * (((int64_t)H * W + 31) / 32 + 2 * guard);
      UnfoldArgs u;
      u.x = x; u.planes = planes; u.pw = (H * W + 31) / 32;
      u.row_bits = row_bits; u.col_bits = col_bits; u.colsum = colsum;
      u.row_words = fqt1_packed_words(Ki); u.col_words = fqt1_packed_words(Mi);
      u.C = C; u.H = H; u.W = W; u.kh = kh; u.kw = kw; u.stride = stride; u.pad = pad; u.Wo = Wo;
      u.M = (int)Mi; u.K = (int)Ki; u.khw = kh * kw; u.HWo = Ho * Wo; u.tm = tm;
      u.guard = guard; u.same = same ? 1 : 0;
      u.div_khw = FastDiv((uint32_t)(kh * kw)); u.div_kw = FastDiv((uint32_t)kw);
      u.div_hwo = FastDiv((uint32_t)(Ho * Wo)); u.div_wo = FastDiv((uint32_t)Wo);
      const int64_t row_tiles = (Mi + tm - 1) / tm, word_tiles = (u.row_words + 7) / 8;
      static std::atomic<uint64_t> attr{0};
      FQT1_CUDA_TRY(smem_attr_once((const void*)unfold_bits_kernel, kUnfoldMaxStreamWords * 4, attr));
      if (colsum) FQT1_CUDA_TRY(cudaMemsetAsync(colsum, 0, sizeof(int32_t) * Ki, s));
      launch_k(unfold_bits_kernel, dim3((unsigned)word_tiles, (unsigned)row_tiles), dim3(256), (size_t)words * 4, s, u);
      fqt1_count_launches(1);
      FQT1_CUDA_TRY(cudaGetLastError());
      const int64_t written = row_tiles * (tm / 32);
      if (col_bits && u.col_words > written) {
        const int64_t n = Ki * (u.col_words - written);
        launch_k(zero_col_pad_kernel, dim3((unsigned)((n + 255) / 256)), dim3(256), 0, s, col_bits, Ki, u.col_words, written);
        fqt1_count_launches(1);
        FQT1_CUDA_TRY(cudaGetLastError());
      }
      return FQT1_OK;
    }
  }
  if (!x) return FQT1_ERR_UNSUPPORTED;  // the gather path reads x itself
  Im2colLoader L;
  L.x = x; L.rows = (int64_t)N * Ho * Wo; L.cols = (int64_t)C * kh * kw;
  L.H = H; L.W = W; L.stride = stride; L.pad = pad; L.CHW = C * H * W; L.HW = H * W;
  L.div_hw_out = FastDiv((uint32_t)(Ho * Wo)); L.div_wo = FastDiv((uint32_t)Wo);
  L.div_khw = FastDiv((uint32_t)(kh * kw)); L.div_kw = FastDiv((uint32_t)kw);
  return launch_pack(L, row_bits, col_bits, colsum, s);
}

extern "C" fqt1_status fqt1_pack_pixels(const float* x, int32_t N, int32_t C, int32_t H, int32_t W, uint32_t* x_pix,
                                        void* stream) {
  if (!x || !x_pix || N < 1 || C < 1 || H < 1 || W < 1) return FQT1_ERR_INVALID_ARG;
  if (C % (32 * kPixBlocks) != 0) return FQT1_ERR_UNSUPPORTED;
  if (!aligned16(x_pix)) return FQT1_ERR_MISALIGNED;
  const int64_t P = (int64_t)N * H * W;
  if ((int64_t)N * C * H * W >= (1ll << 31) || (P + 31) / 32 >= (1ll << 31)) return FQT1_ERR_UNSUPPORTED;
  const int64_t words = fqt1_packed_words(C);
  FQT1_CUDA_TRY(launch_k(pack_pixels_kernel, dim3((unsigned)((P + 31) / 32), (unsigned)(C / (32 * kPixBlocks))),
                         dim3(32 * kPixBlocks), 0, (cudaStream_t)stream, x, P, (int)C, H * W,
                         FastDiv((uint32_t)(H * W)), words, x_pix));
  fqt1_count_launches(1);
  return FQT1_OK;
}

extern "C" fqt1_status fqt1_pack_weight_taps(const float* w, int64_t D, int32_t C, int32_t kh, int32_t kw,
                                             uint32_t* w_taps, void* stream) {
  if (!w || !w_taps || D < 1 || C < 1 || kh < 1 || kw < 1) return FQT1_ERR_INVALID_ARG;
  if (C % 32 != 0) return FQT1_ERR_UNSUPPORTED;
  if (!aligned16(w_taps)) return FQT1_ERR_MISALIGNED;
  const int64_t khw = (int64_t)kh * kw;
  if (D * C * khw >= (1ll << 40) || (D * khw + 7) / 8 >= (1ll << 31)) return FQT1_ERR_UNSUPPORTED;
  const int64_t words = fqt1_packed_words(khw * C);
  FQT1_CUDA_TRY(launch_k(pack_weight_taps_kernel, dim3((unsigned)((D * khw + 7) / 8)), dim3(256), 0,
                         (cudaStream_t)stream, w, D, (int)C, (int)khw, words, w_taps));
  fqt1_count_launches(1);
  return FQT1_OK;
}

extern "C" fqt1_status fqt1_expand_signs_e4m3(const uint32_t* bits, int64_t rows, int64_t n, uint8_t* out,
                                              int64_t ld_out, void* stream) {
  if (!bits || !out || rows < 1 || n < 1 || ld_out < n || ld_out % 16) return FQT1_ERR_INVALID_ARG;
  if (!aligned16(bits) || !aligned16(out)) return FQT1_ERR_MISALIGNED;
  const int64_t threads = rows * (ld_out / 16);
  if ((threads + 255) / 256 >= (1ll << 31)) return FQT1_ERR_UNSUPPORTED;
  FQT1_CUDA_TRY(launch_k(expand_signs_kernel, dim3((unsigned)((threads + 255) / 256)), dim3(256), 0,
                         (cudaStream_t)stream, bits, rows, n, fqt1_packed_words(n), out, ld_out));
  fqt1_count_launches(1);
  return FQT1_OK;
}

extern "C" fqt1_status fqt1_binarize_pack_e4m3(const float* x, int64_t rows, int64_t cols, int64_t ld,
                                               uint32_t* row_bits, uint32_t* col_bits, int32_t* colsum,
                                               uint8_t* row_e4m3, int64_t ld_re, uint8_t* col_e4m3, int64_t ld_ce,
                                               void* stream) {
  if (!x || rows < 1 || cols < 1 || ld < cols) return FQT1_ERR_INVALID_ARG;
  if (!row_bits && !col_bits && !colsum && !row_e4m3 && !col_e4m3) return FQT1_ERR_INVALID_ARG;
  if ((row_e4m3 && (ld_re < cols || ld_re % 16)) || (col_e4m3 && (ld_ce < rows || ld_ce % 16)))
    return FQT1_ERR_INVALID_ARG;
  if (!aligned16(x) || (row_bits && !aligned16(row_bits)) || (col_bits && !aligned16(col_bits)) ||
      (colsum && !aligned16(colsum)) || (row_e4m3 && !aligned16(row_e4m3)) || (col_e4m3 && !aligned16(col_e4m3)))
    return FQT1_ERR_MISALIGNED;
  const int64_t bands = (rows + 31) / 32;
  if (bands > 65535) return FQT1_ERR_UNSUPPORTED;
  if (cols % 4 != 0 || ld % 4 != 0) {
    // no shared-memory tile for these rows: the packed signs, then their byte expansion
    uint32_t* rb = row_bits;
    uint32_t* cbits = col_bits;
    if ((row_e4m3 && !rb) || (col_e4m3 && !cbits)) return FQT1_ERR_INVALID_ARG;
    fqt1_status st = fqt1_binarize_pack(x, rows, cols, ld, rb, cbits, colsum, stream);
    if (st != FQT1_OK) return st;
    if (row_e4m3 && (st = fqt1_expand_signs_e4m3(rb, rows, cols, row_e4m3, ld_re, stream)) != FQT1_OK) return st;
    if (col_e4m3 && (st = fqt1_expand_signs_e4m3(cbits, cols, rows, col_e4m3, ld_ce, stream)) != FQT1_OK) return st;
    return FQT1_OK;
  }
  cudaStream_t s = (cudaStream_t)stream;
  const int64_t row_words = fqt1_packed_words(cols), col_words = fqt1_packed_words(rows);
  if (colsum) FQT1_CUDA_TRY(cudaMemsetAsync(colsum, 0, sizeof(int32_t) * cols, s));
  FQT1_CUDA_TRY(launch_k(pack_tile_kernel, dim3((unsigned)((cols + 32 * kPackTileWarps - 1) / (32 * kPackTileWarps)),
                                                (unsigned)bands),
                         dim3(32 * kPackTileWarps), 0, s, x, rows, cols, ld, row_bits, row_words, col_bits, col_words,
                         colsum, row_e4m3, ld_re, col_e4m3, ld_ce));
  fqt1_count_launches(1);
  if (col_bits && col_words > bands) {
    const int64_t n = cols * (col_words - bands);
    FQT1_CUDA_TRY(launch_k(zero_col_pad_kernel, dim3((unsigned)((n + 255) / 256)), dim3(256), 0, s, col_bits, cols,
                           col_words, bands));
    fqt1_count_launches(1);
  }
  return FQT1_OK;
}

extern "C" fqt1_status fqt1_im2col(const float* x, int32_t N, int32_t C, int32_t H, int32_t W, int32_t kh,
                                   int32_t kw, int32_t stride, int32_t pad, uint32_t* row_bits, uint32_t* col_bits,
                                   int32_t* colsum, void* stream) {
  if (!x) return FQT1_ERR_INVALID_ARG;
  return im2col_impl(x, nullptr, N, C, H, W, kh, kw, stride, pad, row_bits, col_bits, colsum, stream);
}

extern "C" fqt1_status fqt1_im2col_e4m3(const float* x, int32_t N, int32_t C, int32_t H, int32_t W, int32_t kh,
                                        int32_t kw, int32_t stride, int32_t pad, uint8_t* x_row, int64_t ld_row,
                                        uint8_t* x_col, int64_t ld_col, int32_t* colsum, void* stream) {
  if (!x || (!x_row && !x_col)) return FQT1_ERR_INVALID_ARG;
  return im2col_impl(x, nullptr, N, C, H, W, kh, kw, stride, pad, nullptr, nullptr, colsum, stream, x_row, ld_row,
                     x_col, ld_col);
}

extern "C" fqt1_status fqt1_im2col_planes(const uint32_t* planes, int32_t N, int32_t C, int32_t H, int32_t W,
                                          int32_t kh, int32_t kw, int32_t stride, int32_t pad, uint32_t* row_bits,
                                          uint32_t* col_bits, int32_t* colsum, void* stream) {
  if (!planes) return FQT1_ERR_INVALID_ARG;
  return im2col_impl(nullptr, planes, N, C, H, W, kh, kw, stride, pad, row_bits, col_bits, colsum, stream);
}

extern "C" fqt1_status fqt1_pack_planes(const float* x, int32_t N, int32_t C, int32_t H, int32_t W, uint32_t* planes,
                                        void* stream) {
  if (!x || !planes || N < 1 || C < 1 || H < 1 || W < 1) return FQT1_ERR_INVALID_ARG;
  if ((int64_t)N * C * H * W >= (1ll << 31)) return FQT1_ERR_UNSUPPORTED;
  const int pw = (H * W + 31) / 32;
  if (H * W < 32 && 32 % (H * W) == 0) {  // several planes per 32 floats
    const int64_t total = (int64_t)N * C * H * W, chunks = (total + 31) / 32;
    const unsigned blocks = (unsigned)std::min<int64_t>((chunks + 63) / 64, 152 * 16);
    FQT1_CUDA_TRY(launch_k(pack_planes_small_kernel, dim3(blocks), dim3(256), 0, (cudaStream_t)stream, x, total,
                           H * W, planes));
    fqt1_count_launches(1);
    return FQT1_OK;
  }
  const int64_t units = (int64_t)N * C * ((pw + 7) / 8);
  const unsigned blocks = (unsigned)std::min<int64_t>((units + 7) / 8, 152 * 16);
  FQT1_CUDA_TRY(launch_k(pack_planes_nchw_kernel, dim3(blocks), dim3(256), 0, (cudaStream_t)stream, x,
                         (int64_t)N * C, H * W, pw, planes));
  fqt1_count_launches(1);
  return FQT1_OK;
}

extern "C" int32_t fqt1_im2col_path(int32_t N, int32_t C, int32_t H, int32_t W, int32_t kh, int32_t kw,
                                    int32_t stride, int32_t pad) {
  if (N < 1 || C < 1 || H < 1 || W < 1 || kh < 1 || kw < 1 || stride < 1 || pad < 0) return -1;
  const int64_t Ho = conv_extent(H, kh, stride, pad), Wo = conv_extent(W, kw, stride, pad);
  if (Ho < 1 || Wo < 1) return -1;
  if ((int64_t)N * C * H * W >= (1ll << 31) || N * Ho * Wo >= (1ll << 31)) return -1;  // fqt1_im2col refuses these
  if (unfold_same_fits(N, C, H, W, kh, kw, stride, pad)) return 2;
  if (pointwise_conv(kh, kw, pad) && (int64_t)N * ((H - 1) / stride + 1) * ((W - 1) / stride + 1) < (1ll << 31))
    return 3;
  return unfold_bits_tm(N, C, H, W, kh, kw, stride, pad) ? 1 : 0;
}

extern "C" fqt1_status fqt1_pack_planes_nhwc(const float* x, int32_t N, int32_t C, int32_t H, int32_t W,
                                             uint32_t* planes, void* stream) {
  if (!x || !planes || N < 1 || C < 1 || H < 1 || W < 1) return FQT1_ERR_INVALID_ARG;
  if (C % 32 != 0) return FQT1_ERR_UNSUPPORTED;
  if (!aligned16(x)) return FQT1_ERR_MISALIGNED;
  if ((int64_t)N * C * H * W >= (1ll << 31)) return FQT1_ERR_UNSUPPORTED;
  const int pw = (H * W + 31) / 32;
  const int64_t units = (int64_t)N * pw * (C / 32);
  const unsigned blocks = (unsigned)std::min<int64_t>((units + 7) / 8, 152 * 16);
  FQT1_CUDA_TRY(launch_k(pack_planes_nhwc_kernel, dim3(blocks), dim3(256), 0, (cudaStream_t)stream, x, N, C, H * W,
                         pw, planes));
  fqt1_count_launches(1);
  return FQT1_OK;
}
