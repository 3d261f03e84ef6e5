// CUDA-core integer GEMMs on packed signs and bit-planes (App. C, "binary
// multiplication" and Fig. "1-bitmm"): the forward XNOR-popcount product and
// the AND-popcount product of b-bit gradient codes with +-1 signs.  These
// are the small-problem path; large problems go to the tensor-core kernels.
#include "gemm.cuh"

namespace fqt1 {

constexpr int kST = 64;     // output tile (rows and columns)
constexpr int kSW = 8;      // packed words per K step (256 elements)

// acc[m, n] = sum_k sa[m, k] sb[n, k] = K - 2 popc(xor) over the packed words.
__global__ void __launch_bounds__(256) xnor_gemm_simt_kernel(const uint32_t* __restrict__ A,
                                                             const uint32_t* __restrict__ B, int64_t M, int64_t N,
                                                             int64_t K, int64_t ldw, const float* __restrict__ gamma,
                                                             const float* __restrict__ bias,
                                                             int32_t* __restrict__ acc_out, float* __restrict__ y) {
  FQT1_PDL_WAIT();
  FQT1_PDL_TRIGGER();
  __shared__ uint32_t As[kSW][kST + 1], Bs[kSW][kST + 1];
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  const int64_t m0 = (int64_t)blockIdx.y * kST, n0 = (int64_t)blockIdx.x * kST;
  int pc[4][4] = {};
  for (int64_t w0 = 0; w0 < ldw; w0 += kSW) {
    for (int idx = threadIdx.x; idx < kST * kSW; idx += 256) {
      const int r = idx / kSW, q = idx % kSW;
      const int64_t w = w0 + q;
      As[q][r] = (m0 + r < M && w < ldw) ? __ldg(A + (m0 + r) * ldw + w) : 0u;
      Bs[q][r] = (n0 + r < N && w < ldw) ? __ldg(B + (n0 + r) * ldw + w) : 0u;
    }
    __syncthreads();
#pragma unroll
    for (int q = 0; q < kSW; ++q) {
      uint32_t a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) { a[i] = As[q][ty * 4 + i]; b[i] = Bs[q][tx * 4 + i]; }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) pc[i][j] += __popc(a[i] ^ b[j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int64_t m = m0 + ty * 4 + i;
    if (m >= M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int64_t n = n0 + tx * 4 + j;
      if (n >= N) continue;
      const int32_t v = (int32_t)K - 2 * pc[i][j];
      if (acc_out) acc_out[m * N + n] = v;
      if (y) {
        const float g = __fmul_rn(__ldg(gamma + n), __int2float_rn(v));
        y[m * N + n] = bias ? __fadd_rn(g, __ldg(bias + n)) : g;
      }
    }
  }
}

// out[r, s] = sum_j q[r, j] sgn[s, j]: q uint8 codes of `bits` bits (rows r < *count * rows_per_count),
// sgn packed +-1 signs.  Per bit-plane p: sum_j a_j s_j = 2 popc(a & w) - popc(a), merged by 2^p.
template <int BITS>
__global__ void __launch_bounds__(256) codes_gemm_simt_kernel(const uint8_t* __restrict__ Q, int64_t ldq,
                                                              const int32_t* __restrict__ count,
                                                              int64_t rows_per_count,
                                                              const uint32_t* __restrict__ S, int64_t lds,
                                                              int64_t n_s, int64_t L, int32_t* __restrict__ out,
                                                              int64_t ldo) {
  FQT1_PDL_WAIT();
  FQT1_PDL_TRIGGER();
  __shared__ uint32_t Ap[BITS][kSW][kST + 1], Bs[kSW][kST + 1];
  const int64_t n_r = (int64_t)__ldg(count) * rows_per_count;
  const int64_t r0 = (int64_t)blockIdx.y * kST, s0 = (int64_t)blockIdx.x * kST;
  if (r0 >= n_r) return;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  int acc[4][4] = {};
  for (int64_t w0 = 0; w0 < lds; w0 += kSW) {
    for (int rr = 0; rr < 8; ++rr) {
      const int r = warp * 8 + rr;
      const int64_t row = r0 + r;
#pragma unroll
      for (int q = 0; q < kSW; ++q) {
        const int64_t j = (w0 + q) * 32 + lane;
        const uint32_t code = (row < n_r && j < L) ? (uint32_t)__ldg(Q + row * ldq + j) : 0u;
#pragma unroll
        for (int p = 0; p < BITS; ++p) {
          const uint32_t word = __ballot_sync(0xFFFFFFFFu, (code >> p) & 1u);
          if (lane == 0) Ap[p][q][r] = word;
        }
      }
    }
    for (int idx = threadIdx.x; idx < kST * kSW; idx += 256) {
      const int r = idx / kSW, q = idx % kSW;
      const int64_t w = w0 + q;
      Bs[q][r] = (s0 + r < n_s && w < lds) ? __ldg(S + (s0 + r) * lds + w) : 0u;
    }
    __syncthreads();
#pragma unroll 2
    for (int q = 0; q < kSW; ++q) {
      uint32_t b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) b[i] = Bs[q][tx * 4 + i];
#pragma unroll
      for (int p = 0; p < BITS; ++p) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const uint32_t a = Ap[p][q][ty * 4 + i];
          const int pa = __popc(a);
#pragma unroll
          for (int j = 0; j < 4; ++j) acc[i][j] += (2 * __popc(a & b[j]) - pa) << p;
        }
      }
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int64_t r = r0 + ty * 4 + i;
    if (r >= n_r) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int64_t s = s0 + tx * 4 + j;
      if (s < n_s) out[r * ldo + s] = acc[i][j];
    }
  }
}

cudaError_t launch_xnor_gemm_simt(const uint32_t* A, const uint32_t* B, int64_t M, int64_t N, int64_t K,
                                  const float* gamma, const float* bias, int32_t* acc, float* y, cudaStream_t s) {
  const int64_t ldw = fqt1_packed_words(K);
  dim3 grid((unsigned)((N + kST - 1) / kST), (unsigned)((M + kST - 1) / kST));
  launch_k(xnor_gemm_simt_kernel, dim3(grid), dim3(256), 0, s, A, B, M, N, K, ldw, gamma, bias, acc, y);
  fqt1_count_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_codes_gemm_simt(int bits, const uint8_t* Q, int64_t ldq, const int32_t* count,
                                   int64_t rows_per_count, int64_t max_rows, const uint32_t* S, int64_t n_s,
                                   int64_t L, int32_t* out, int64_t ldo, cudaStream_t s) {
  const int64_t lds = fqt1_packed_words(L);
  dim3 grid((unsigned)((n_s + kST - 1) / kST), (unsigned)((max_rows + kST - 1) / kST));
  switch (bits) {
    case 1: launch_k(codes_gemm_simt_kernel<1>, dim3(grid), dim3(256), 0, s, Q, ldq, count, rows_per_count, S, lds, n_s, L, out, ldo); break;
    case 2: launch_k(codes_gemm_simt_kernel<2>, dim3(grid), dim3(256), 0, s, Q, ldq, count, rows_per_count, S, lds, n_s, L, out, ldo); break;
    case 4: launch_k(codes_gemm_simt_kernel<4>, dim3(grid), dim3(256), 0, s, Q, ldq, count, rows_per_count, S, lds, n_s, L, out, ldo); break;
    default: launch_k(codes_gemm_simt_kernel<8>, dim3(grid), dim3(256), 0, s, Q, ldq, count, rows_per_count, S, lds, n_s, L, out, ldo); break;
  }
  fqt1_count_launches(1);
  return cudaGetLastError();
}

}  // namespace fqt1
