// Sign + pack kernels: the row / column encoders of App. C (Algorithm 2) and the
// Unfolder fused with them.  One pass over the input writes both packings and
// the column sums of the signs.
#include "common.cuh"

namespace fqt1 {

// A CTA covers Loader::kRows rows (32 or 64) x 256 columns (8 packed words) of the
// logical matrix.  Warp w packs rows w, w+8, ... along the columns with __ballot_sync;
// the row words of each 32-column slab then give, read bit-wise per column, the
// column-packed words of those rows (one per 32 rows).
constexpr int kPackWordsPerCta = 8;

// A loader splits element (r, c) into a per-row part and a per-column part, so that a
// warp computes its row part once per row and a lane its column parts once per CTA.
struct DenseLoader {
  static constexpr int kRows = 32;  // rows per CTA
  const float* x;
  int64_t rows, cols, ld;
  struct Col { int64_t c; bool ok; };
  struct Row { const float* p; bool ok; };
  __device__ __forceinline__ Col col(int64_t c) const { return {c, c < cols}; }
  __device__ __forceinline__ Row row(int64_t r) const { return {x + r * ld, r < rows}; }
  __device__ __forceinline__ float load(const Row& r, const Col& c) const {
    return (r.ok && c.ok) ? __ldg(r.p + c.c) : 0.0f;
  }
};

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

// Column-packed words past ceil(rows/32) (the alignment padding) are zero.
__global__ void zero_col_pad_kernel(uint32_t* col_bits, int64_t cols, int64_t col_words, int64_t first_pad) {
  const int64_t npad = col_words - first_pad;
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i < cols * npad) col_bits[(i / npad) * col_words + first_pad + (i % npad)] = 0u;
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
  pack_kernel<Loader><<<grid, 256, 0, s>>>(L, row_bits, row_words, col_bits, col_words, colsum);
  fqt1_count_launches(1);
  FQT1_CUDA_TRY(cudaGetLastError());
  if (col_bits && col_words > col_words_written) {
    const int64_t n = L.cols * (col_words - col_words_written);
    zero_col_pad_kernel<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(col_bits, L.cols, col_words,
                                                                    col_words_written);
    fqt1_count_launches(1);
    FQT1_CUDA_TRY(cudaGetLastError());
  }
  return FQT1_OK;
}

}  // namespace fqt1

using namespace fqt1;

static bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

extern "C" fqt1_status fqt1_binarize_pack(const float* x, int64_t rows, int64_t cols, int64_t ld,
                                          uint32_t* row_bits, uint32_t* col_bits, int32_t* colsum,
                                          void* stream) {
  if (!x || rows < 1 || cols < 1 || ld < cols) return FQT1_ERR_INVALID_ARG;
  if (!row_bits && !col_bits && !colsum) return FQT1_ERR_INVALID_ARG;
  if (!aligned16(x) || (row_bits && !aligned16(row_bits)) || (col_bits && !aligned16(col_bits)) ||
      (colsum && !aligned16(colsum)))
    return FQT1_ERR_MISALIGNED;
  DenseLoader L{x, rows, cols, ld};
  return launch_pack(L, row_bits, col_bits, colsum, (cudaStream_t)stream);
}

extern "C" fqt1_status fqt1_im2col(const float* x, int32_t N, int32_t C, int32_t H, int32_t W, int32_t kh,
                                   int32_t kw, int32_t stride, int32_t pad, uint32_t* row_bits, uint32_t* col_bits,
                                   int32_t* colsum, void* stream) {
  if (!x || N < 1 || C < 1 || H < 1 || W < 1 || kh < 1 || kw < 1 || stride < 1 || pad < 0)
    return FQT1_ERR_INVALID_ARG;
  if (!row_bits && !col_bits && !colsum) return FQT1_ERR_INVALID_ARG;
  const int Ho = (H + 2 * pad - kh) / stride + 1, Wo = (W + 2 * pad - kw) / stride + 1;
  if (H + 2 * pad < kh || W + 2 * pad < kw || Ho < 1 || Wo < 1) return FQT1_ERR_INVALID_ARG;
  if (!aligned16(x) || (row_bits && !aligned16(row_bits)) || (col_bits && !aligned16(col_bits)) ||
      (colsum && !aligned16(colsum)))
    return FQT1_ERR_MISALIGNED;
  if ((int64_t)N * C * H * W >= (1ll << 31) || (int64_t)N * Ho * Wo >= (1ll << 31)) return FQT1_ERR_UNSUPPORTED;
  Im2colLoader L;
  L.x = x; L.rows = (int64_t)N * Ho * Wo; L.cols = (int64_t)C * kh * kw;
  L.H = H; L.W = W; L.stride = stride; L.pad = pad; L.CHW = C * H * W; L.HW = H * W;
  L.div_hw_out = FastDiv((uint32_t)(Ho * Wo)); L.div_wo = FastDiv((uint32_t)Wo);
  L.div_khw = FastDiv((uint32_t)(kh * kw)); L.div_kw = FastDiv((uint32_t)kw);
  return launch_pack(L, row_bits, col_bits, colsum, (cudaStream_t)stream);
}
