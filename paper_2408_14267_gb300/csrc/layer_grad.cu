// Gradients of a layer's own parameters and the clipped straight-through estimator.
//
// The layer computes y = (sign(x) sign(W)^T) (.) Gamma + bias (Sec. 5.1, the scaling factor
// Gamma in R^D shared by weights and activations; a bias is an extension, the paper's
// Algorithm 1 omits it).  With acc = sign(x) sign(W)^T the int32 forward accumulators:
//   dGamma[j] = sum_m gY[m, j] acc[m, j],   dbias[j] = sum_m gY[m, j].
// Both sums run in a fixed order (fp32 within chunks of kChunkRows rows, float64 over the
// chunks), so the results do not depend on the launch.
//
// The straight-through estimator (cited in Sec. 3.1 for QAT) passes the gradient of sign()
// through unchanged by default; its clipped form keeps it only where |x| <= t.
#include <algorithm>

#include "common.cuh"

namespace fqt1 {

constexpr int kChunkRows = 256;  // rows of gY per partial sum
constexpr int kGradCols = 32;    // columns per CTA (one per lane)
constexpr int kRowLanes = 8;     // warps of a CTA; warp w takes rows w, w + 8, ... of a chunk

// part[c][j] and part[chunks + c][j] = the fp32 sums of gY acc and gY over rows c kChunkRows ..
// (c + 1) kChunkRows - 1: each warp sums its rows in order, then the 8 warp sums are added in
// warp order.
template <bool ACC>
__global__ void __launch_bounds__(kGradCols * kRowLanes) scale_bias_partial_kernel(
    const float* __restrict__ gy, const int32_t* __restrict__ acc, int64_t M, int64_t D, int64_t chunks,
    float* __restrict__ part) {
  FQT1_PDL_WAIT();
  FQT1_PDL_TRIGGER();
  __shared__ float sg_s[kRowLanes][kGradCols], sb_s[kRowLanes][kGradCols];
  const int lane = threadIdx.x & 31, rl = threadIdx.x >> 5;
  const int64_t j = (int64_t)blockIdx.x * kGradCols + lane;
  const int64_t jc = min(j, D - 1);
  const int64_t c = blockIdx.y, r0 = c * kChunkRows + rl;
  float sg = 0.f, sb = 0.f;
#pragma unroll 1
  for (int i0 = 0; i0 < kChunkRows / kRowLanes; i0 += 8) {
    // 8 rows in flight (unconditional loads from clamped rows, masked below)
    float g[8];
    int32_t q[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int64_t r = min(r0 + (int64_t)kRowLanes * (i0 + u), M - 1);
      g[u] = __ldg(gy + r * D + jc);
      q[u] = ACC ? __ldg(acc + r * D + jc) : 0;
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      if (r0 + (int64_t)kRowLanes * (i0 + u) >= M) break;
      sg = __fadd_rn(sg, __fmul_rn(g[u], (float)q[u]));
      sb = __fadd_rn(sb, g[u]);
    }
  }
  sg_s[rl][lane] = sg;
  sb_s[rl][lane] = sb;
  __syncthreads();
  if (rl == 0 && j < D) {
    float tg = 0.f, tb = 0.f;
#pragma unroll
    for (int w = 0; w < kRowLanes; ++w) {
      tg = __fadd_rn(tg, sg_s[w][lane]);
      tb = __fadd_rn(tb, sb_s[w][lane]);
    }
    part[c * D + j] = tg;
    part[(chunks + c) * D + j] = tb;
  }
}

// dgamma[j], dbias[j]: warp w adds chunks w, w + 8, ... in float64, then the 8 warp sums are
// added in warp order.
__global__ void __launch_bounds__(kGradCols * kRowLanes) scale_bias_final_kernel(
    const float* __restrict__ part, int64_t D, int64_t chunks, float* __restrict__ dgamma, float* __restrict__ dbias) {
  FQT1_PDL_WAIT();
  FQT1_PDL_TRIGGER();
  __shared__ double sg_s[kRowLanes][kGradCols], sb_s[kRowLanes][kGradCols];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int64_t j = (int64_t)blockIdx.x * kGradCols + lane;
  const int64_t jc = min(j, D - 1);
  double sg = 0.0, sb = 0.0;
  for (int64_t c = w; c < chunks; c += kRowLanes) {
    sg += (double)__ldg(part + c * D + jc);
    sb += (double)__ldg(part + (chunks + c) * D + jc);
  }
  sg_s[w][lane] = sg;
  sb_s[w][lane] = sb;
  __syncthreads();
  if (w == 0 && j < D) {
    double tg = 0.0, tb = 0.0;
#pragma unroll
    for (int u = 0; u < kRowLanes; ++u) {
      tg += sg_s[u][lane];
      tb += sb_s[u][lane];
    }
    if (dgamma) dgamma[j] = (float)tg;
    if (dbias) dbias[j] = (float)tb;
  }
}

__global__ void __launch_bounds__(256) ste_clip_kernel(const float* __restrict__ x, float* __restrict__ dx,
                                                       int64_t n, float t) {
  FQT1_PDL_WAIT();
  FQT1_PDL_TRIGGER();
  const int64_t n4 = n / 4;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += stride) {
    const float4 v = __ldg(reinterpret_cast<const float4*>(x) + i);
    float4 g = reinterpret_cast<float4*>(dx)[i];
    g.x = fabsf(v.x) <= t ? g.x : 0.f;
    g.y = fabsf(v.y) <= t ? g.y : 0.f;
    g.z = fabsf(v.z) <= t ? g.z : 0.f;
    g.w = fabsf(v.w) <= t ? g.w : 0.f;
    reinterpret_cast<float4*>(dx)[i] = g;
  }
  for (int64_t i = 4 * n4 + (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride)
    dx[i] = fabsf(x[i]) <= t ? dx[i] : 0.f;
}

}  // namespace fqt1

using namespace fqt1;

static bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

extern "C" size_t fqt1_scale_bias_workspace(int64_t M, int64_t D) {
  if (M < 1 || D < 1) return 0;
  return (size_t)(2 * ((M + kChunkRows - 1) / kChunkRows) * D) * sizeof(float);
}

extern "C" fqt1_status fqt1_scale_bias_grad(const float* gy, const int32_t* acc, int64_t M, int64_t D,
                                            float* dgamma, float* dbias, void* ws, size_t ws_bytes, void* stream) {
  if (!gy || M < 1 || D < 1 || (!dgamma && !dbias) || (dgamma && !acc)) return FQT1_ERR_INVALID_ARG;
  if (!aligned16(gy) || (acc && !aligned16(acc)) || (dgamma && !aligned16(dgamma)) || (dbias && !aligned16(dbias)))
    return FQT1_ERR_MISALIGNED;
  const int64_t chunks = (M + kChunkRows - 1) / kChunkRows;
  if (!ws || ws_bytes < fqt1_scale_bias_workspace(M, D)) return FQT1_ERR_WORKSPACE;
  if (!aligned16(ws)) return FQT1_ERR_MISALIGNED;
  if (chunks > 65535) return FQT1_ERR_UNSUPPORTED;
  cudaStream_t s = (cudaStream_t)stream;
  float* part = static_cast<float*>(ws);
  const unsigned gx = (unsigned)((D + kGradCols - 1) / kGradCols);
  const dim3 block(kGradCols * kRowLanes);
  if (dgamma)
    FQT1_CUDA_TRY(launch_k(scale_bias_partial_kernel<true>, dim3(gx, (unsigned)chunks), block, 0, s, gy, acc, M, D,
                           chunks, part));
  else
    FQT1_CUDA_TRY(launch_k(scale_bias_partial_kernel<false>, dim3(gx, (unsigned)chunks), block, 0, s, gy, acc, M, D,
                           chunks, part));
  fqt1_count_launches(1);
  FQT1_CUDA_TRY(launch_k(scale_bias_final_kernel, dim3(gx), block, 0, s, part, D, chunks, dgamma, dbias));
  fqt1_count_launches(1);
  return FQT1_OK;
}

extern "C" fqt1_status fqt1_ste_clip(const float* x, float* dx, int64_t n, float t, void* stream) {
  if (!x || !dx || n < 1 || !(t >= 0.0f)) return FQT1_ERR_INVALID_ARG;
  if (!aligned16(x) || !aligned16(dx)) return FQT1_ERR_MISALIGNED;
  const int64_t blocks = std::min<int64_t>((n / 4 + 255) / 256 + 1, 4096);
  FQT1_CUDA_TRY(launch_k(ste_clip_kernel, dim3((unsigned)blocks), dim3(256), 0, (cudaStream_t)stream, x, dx, n, t));
  fqt1_count_launches(1);
  return FQT1_OK;
}
