// Sign + pack kernels: the row / column encoders of App. C (Algorithm 2) and the
// Unfolder fused with them.  One pass over the input writes both packings and
// the column sums of the signs.
#include "common.cuh"

namespace fqt1 {

// A CTA covers 32 rows x 256 columns (8 packed words) of the logical matrix.
// Warp w packs rows w, w+8, w+16, w+24 along the columns with __ballot_sync;
// the 32 row words of each 32-column slab then give, read bit-wise per
// column, the column-packed word of those 32 rows.
constexpr int kPackRows = 32;
constexpr int kPackWordsPerCta = 8;

struct DenseLoader {
  const float* x;
  int64_t rows, cols, ld;
  __device__ __forceinline__ bool valid(int64_t r, int64_t c) const { return r < rows && c < cols; }
  __device__ __forceinline__ float load(int64_t r, int64_t c) const { return __ldg(x + r * ld + c); }
};

// Element (m, k) of the unfolded matrix X_u = Unfolder(x); outside the image it is 0.
struct Im2colLoader {
  const float* x;
  int64_t rows, cols;  // M = N*Ho*Wo, K = C*kh*kw
  int C, H, W, kh, kw, stride, pad, Ho, Wo;
  __device__ __forceinline__ bool valid(int64_t r, int64_t c) const { return r < rows && c < cols; }
  __device__ __forceinline__ float load(int64_t m, int64_t k) const {
    const int64_t hw = (int64_t)Ho * Wo;
    const int64_t n = m / hw;
    const int rem = (int)(m - n * hw);
    const int oh = rem / Wo, ow = rem - (rem / Wo) * Wo;
    const int khw = kh * kw;
    const int c = (int)(k / khw);
    const int t = (int)(k - (int64_t)c * khw);
    const int i = t / kw, j = t - (t / kw) * kw;
    const int h = oh * stride - pad + i, w = ow * stride - pad + j;
    if (h < 0 || h >= H || w < 0 || w >= W) return 0.0f;
    return __ldg(x + (((n * C + c) * (int64_t)H + h) * W + w));
  }
};

template <class Loader>
__global__ void __launch_bounds__(256) pack_kernel(Loader L, uint32_t* __restrict__ row_bits, int64_t row_words,
                                                   uint32_t* __restrict__ col_bits, int64_t col_words,
                                                   int32_t* __restrict__ colsum) {
  __shared__ uint32_t rw[kPackRows][kPackWordsPerCta];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t r0 = (int64_t)blockIdx.y * kPackRows;
  const int64_t w0 = (int64_t)blockIdx.x * kPackWordsPerCta;
  for (int rr = warp; rr < kPackRows; rr += 8) {
    const int64_t r = r0 + rr;
    float v[kPackWordsPerCta];
#pragma unroll
    for (int q = 0; q < kPackWordsPerCta; ++q) {
      const int64_t c = (w0 + q) * 32 + lane;
      v[q] = L.valid(r, c) ? L.load(r, c) : 0.0f;
    }
#pragma unroll
    for (int q = 0; q < kPackWordsPerCta; ++q) {
      const int64_t c = (w0 + q) * 32 + lane;
      const uint32_t word = __ballot_sync(0xFFFFFFFFu, L.valid(r, c) && v[q] > 0.0f);
      if (lane == 0) rw[rr][q] = word;
    }
  }
  __syncthreads();
  // Row-packed output: word (r, w0 + q).
  if (row_bits) {
    const int rr = threadIdx.x >> 3, q = threadIdx.x & 7;
    const int64_t r = r0 + rr, w = w0 + q;
    if (r < L.rows && w < row_words) row_bits[r * row_words + w] = rw[rr][q];
  }
  // Column-packed output: word (c, blockIdx.y) holds rows r0..r0+31 of column c.
  const int q = threadIdx.x >> 5;
  const int64_t c = (w0 + q) * 32 + lane;
  if (c < L.cols) {
    uint32_t cw = 0;
#pragma unroll
    for (int rr = 0; rr < kPackRows; ++rr) cw |= ((rw[rr][q] >> lane) & 1u) << rr;
    if (col_bits) col_bits[c * col_words + blockIdx.y] = cw;
    if (colsum) {
      const int64_t nvalid = min((int64_t)kPackRows, L.rows - r0);
      if (nvalid > 0) atomicAdd(colsum + c, 2 * __popc(cw) - (int)nvalid);
    }
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
  const int64_t row_tiles = (L.rows + kPackRows - 1) / kPackRows;
  const int64_t word_tiles = (row_words + kPackWordsPerCta - 1) / kPackWordsPerCta;
  if (row_tiles > 65535) return FQT1_ERR_UNSUPPORTED;
  if (colsum) FQT1_CUDA_TRY(cudaMemsetAsync(colsum, 0, sizeof(int32_t) * L.cols, s));
  dim3 grid((unsigned)word_tiles, (unsigned)row_tiles);
  pack_kernel<Loader><<<grid, 256, 0, s>>>(L, row_bits, row_words, col_bits, col_words, colsum);
  fqt1_count_launches(1);
  FQT1_CUDA_TRY(cudaGetLastError());
  if (col_bits && col_words > row_tiles) {
    const int64_t n = L.cols * (col_words - row_tiles);
    zero_col_pad_kernel<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(col_bits, L.cols, col_words, row_tiles);
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
  Im2colLoader L{x, (int64_t)N * Ho * Wo, (int64_t)C * kh * kw, C, H, W, kh, kw, stride, pad, Ho, Wo};
  return launch_pack(L, row_bits, col_bits, colsum, (cudaStream_t)stream);
}
