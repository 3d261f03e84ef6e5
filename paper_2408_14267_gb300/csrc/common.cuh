// Device-side helpers shared by the libfqt1 kernels.
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

#include "../../include/fqt1.h"

namespace fqt1 {

constexpr int kStreamSrPsq = 0;      // stochastic rounding, per-sample branch
constexpr int kStreamSrPcq = 1;      // stochastic rounding, per-channel branch
constexpr int kStreamSelSample = 2;  // AGP masks of sample groups
constexpr int kStreamSelChannel = 3; // AGP masks of channels
constexpr int kFixedPointBits = 40;  // fixed-point scale of the group ranges
constexpr int kMaxGroups = 16384;    // one selection CTA sorts at most this many groups

// Philox4x32-10 (Salmon et al., SC'11): 10 rounds of two 32x32->64-bit
// multiplies with the Weyl-bumped key.  Returns the 4 words of one block.
struct U32x4 { uint32_t x, y, z, w; };

__device__ __forceinline__ U32x4 philox4x32_10(uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3, uint32_t k0,
                                               uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const uint32_t hi0 = __umulhi(0xD2511F53u, c0), lo0 = 0xD2511F53u * c0;
    const uint32_t hi1 = __umulhi(0xCD9E8D57u, c2), lo1 = 0xCD9E8D57u * c2;
    const uint32_t n0 = hi1 ^ c1 ^ k0, n2 = hi0 ^ c3 ^ k1;
    c0 = n0; c1 = lo1; c2 = n2; c3 = lo0;
    k0 += 0x9E3779B9u;
    k1 += 0xBB67AE85u;
  }
  return {c0, c1, c2, c3};
}

// The 4 words of counter block `blk` (words 4*blk .. 4*blk+3) of `stream`.
__device__ __forceinline__ U32x4 philox_block(uint64_t seed, uint32_t stream, uint64_t blk) {
  return philox4x32_10((uint32_t)blk, (uint32_t)(blk >> 32), stream, 0u, (uint32_t)seed, (uint32_t)(seed >> 32));
}

__device__ __forceinline__ uint32_t philox_word(uint64_t seed, uint32_t stream, uint64_t index) {
  const U32x4 r = philox_block(seed, stream, index >> 2);
  switch (index & 3) {
    case 0: return r.x;
    case 1: return r.y;
    case 2: return r.z;
    default: return r.w;
  }
}

// Division of 32-bit unsigned n < 2^31 by an invariant d >= 1 with one multiply-high
// (Granlund and Montgomery, "Division by invariant integers using multiplication",
// PLDI'94): with l = ceil(log2 d) and m = floor(2^32 (2^l - d) / d) + 1,
// n / d = (umulhi(n, m) + n) >> l.  The host computes m and l.
struct FastDiv {
  uint32_t d, mul, shr;
  __host__ __device__ FastDiv() : d(1), mul(1), shr(0) {}
  __host__ __device__ explicit FastDiv(uint32_t divisor) : d(divisor), mul(0), shr(0) {
    while (shr < 31 && (1u << shr) < d) ++shr;
    mul = (uint32_t)((((uint64_t)1 << 32) * (((uint64_t)1 << shr) - d)) / d + 1);
  }
  __device__ __forceinline__ uint32_t div(uint32_t n) const { return (__umulhi(n, mul) + n) >> shr; }
};

// Order-preserving map float -> uint32 (so atomicMin/atomicMax give float min/max).
__device__ __forceinline__ uint32_t float_to_ordered(float f) {
  const uint32_t b = __float_as_uint(f);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}
__device__ __forceinline__ float ordered_to_float(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k);
}

// One stochastic rounding of x to [0, B] given inv = B / R (all fp32, round-to-nearest,
// no contraction): q = floor(t) + [u < t - floor(t)], t = (x - Z) * inv, u = (w >> 8) 2^-24.
__device__ __forceinline__ uint32_t sr_code(float x, float z, float inv, float Bf, bool degenerate, uint32_t w) {
  if (degenerate) return 0u;
  const float t = __fmul_rn(__fsub_rn(x, z), inv);
  const float fl = floorf(t);
  const float frac = __fsub_rn(t, fl);
  const float u = __fmul_rn(__uint2float_rn(w >> 8), 5.9604644775390625e-08f);  // 2^-24
  float q = fl + ((u < frac) ? 1.0f : 0.0f);
  q = fminf(fmaxf(q, 0.0f), Bf);
  return (uint32_t)q;
}

}  // namespace fqt1

#define FQT1_CUDA_TRY(expr)                              \
  do {                                                   \
    cudaError_t e__ = (expr);                            \
    if (e__ != cudaSuccess) {                            \
      fqt1_set_cuda_error(e__);                          \
      return FQT1_ERR_CUDA;                              \
    }                                                    \
  } while (0)

// Programmatic dependent launch: every kernel of the library is launched with programmatic
// stream serialization, so its launch and prologue may overlap the tail of the kernel before
// it in the stream.  A kernel calls FQT1_PDL_WAIT() before it touches memory written by
// earlier work (it then sees all of it), and FQT1_PDL_TRIGGER() to let the next kernel start.
#define FQT1_PDL_WAIT() asm volatile("griddepcontrol.wait;" ::: "memory")
#define FQT1_PDL_TRIGGER() asm volatile("griddepcontrol.launch_dependents;" ::: "memory")

namespace fqt1 {
template <typename... KArgs, typename... Args>
inline cudaError_t launch_k(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                            Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// cudaFuncSetAttribute(MaxDynamicSharedMemorySize) applies to the current device only.  A call
// site keeps one bit per device ordinal in `done` for the devices where it has set the
// attribute; the bits are atomic, so host threads may launch concurrently (two threads that
// both set the attribute do no harm).
inline cudaError_t smem_attr_once(const void* fn, int bytes, std::atomic<uint64_t>& done) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = (dev >= 0 && dev < 64) ? (uint64_t)1 << dev : 0;
  if (bit && (done.load(std::memory_order_acquire) & bit)) return cudaSuccess;
  e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess && bit) done.fetch_or(bit, std::memory_order_acq_rel);
  return e;
}

// The same launch as a grid of thread-block clusters of cluster_z CTAs along z.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_k_cluster(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                                    unsigned cluster_z, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = 1;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = cluster_z;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}
}  // namespace fqt1

void fqt1_set_cuda_error(cudaError_t e);
// Replaces the text returned by fqt1_last_cuda_error() with msg.
void fqt1_set_error_text(const char* msg);
// Adds n to the count returned by fqt1_kernel_launches().
void fqt1_count_launches(int n);
