// Datapath probe: throughput of the candidate contraction units on sm_103a and
// exactness of fp32 accumulation of integer-valued fp8 / bf16 products.  The layer
// step's integer products need the fastest unit whose result equals the int32 sum.
//
//   nvcc -gencode arch=compute_103a,code=sm_103a -O3 -std=c++17 -o datapath_probe datapath_probe.cu
//   ./datapath_probe
// (-DPROBE_I8 adds tcgen05 kind::i8, which ptxas rejects for sm_103a.)
#include <cstdio>
#include <cstdint>
#include <cuda_runtime.h>

#define CK(x) do { cudaError_t e = (x); if (e != cudaSuccess) { printf("CUDA %s at %d: %s\n", #x, __LINE__, cudaGetErrorString(e)); return 1; } } while (0)

__global__ void k_b1(int iters, int* out) {
  uint32_t a0 = threadIdx.x * 2654435761u, a1 = a0 ^ 0x55555555u, a2 = a0 + 7, a3 = a0 * 3;
  uint32_t b0 = blockIdx.x * 40503u + 1, b1 = b0 ^ 0xF0F0F0F0u;
  int c[8][4] = {};
  for (int i = 0; i < iters; ++i) {
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      asm volatile("mma.sync.aligned.m16n8k256.row.col.s32.b1.b1.s32.and.popc {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
                   : "+r"(c[j][0]), "+r"(c[j][1]), "+r"(c[j][2]), "+r"(c[j][3])
                   : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
    }
  }
  int s = 0;
  for (int j = 0; j < 8; ++j) s += c[j][0] + c[j][1] + c[j][2] + c[j][3];
  if (s == 0x7fffffff) out[0] = s;
}

__global__ void k_b1x(int iters, int* out) {
  uint32_t a0 = threadIdx.x * 2654435761u, a1 = a0 ^ 0x55555555u, a2 = a0 + 7, a3 = a0 * 3;
  uint32_t b0 = blockIdx.x * 40503u + 1, b1 = b0 ^ 0xF0F0F0F0u;
  int c[8][4] = {};
  for (int i = 0; i < iters; ++i) {
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      asm volatile("mma.sync.aligned.m16n8k256.row.col.s32.b1.b1.s32.xor.popc {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
                   : "+r"(c[j][0]), "+r"(c[j][1]), "+r"(c[j][2]), "+r"(c[j][3])
                   : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
    }
  }
  int s = 0;
  for (int j = 0; j < 8; ++j) s += c[j][0] + c[j][1] + c[j][2] + c[j][3];
  if (s == 0x7fffffff) out[0] = s;
}

__global__ void k_s8(int iters, int* out) {
  uint32_t a0 = threadIdx.x * 2654435761u, a1 = a0 ^ 0x55555555u, a2 = a0 + 7, a3 = a0 * 3;
  uint32_t b0 = blockIdx.x * 40503u + 1, b1 = b0 ^ 0xF0F0F0F0u;
  int c[8][4] = {};
  for (int i = 0; i < iters; ++i) {
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      asm volatile("mma.sync.aligned.m16n8k32.row.col.s32.s8.s8.s32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
                   : "+r"(c[j][0]), "+r"(c[j][1]), "+r"(c[j][2]), "+r"(c[j][3])
                   : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
    }
  }
  int s = 0;
  for (int j = 0; j < 8; ++j) s += c[j][0] + c[j][1] + c[j][2] + c[j][3];
  if (s == 0x7fffffff) out[0] = s;
}

__global__ void k_e4m3(int iters, int* out) {
  uint32_t a0 = 0x38383838u, a1 = 0xB838B838u, a2 = 0x38B838B8u, a3 = 0x38383838u;
  uint32_t b0 = 0x38383838u, b1 = 0xB8B83838u;
  float c[8][4] = {};
  for (int i = 0; i < iters; ++i) {
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      asm volatile("mma.sync.aligned.m16n8k32.row.col.f32.e4m3.e4m3.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
                   : "+f"(c[j][0]), "+f"(c[j][1]), "+f"(c[j][2]), "+f"(c[j][3])
                   : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
    }
  }
  float s = 0;
  for (int j = 0; j < 8; ++j) s += c[j][0] + c[j][1] + c[j][2] + c[j][3];
  if (s == 1.2345f) out[0] = 1;
}

__global__ void k_popc(int iters, int* out) {
  uint32_t a[8], b = blockIdx.x * 2654435761u + threadIdx.x;
  int acc[8] = {};
  for (int j = 0; j < 8; ++j) a[j] = threadIdx.x * (j + 1) * 40503u;
  for (int i = 0; i < iters; ++i) {
#pragma unroll
    for (int j = 0; j < 8; ++j) { acc[j] += __popc(a[j] ^ b); a[j] += 0x9E3779B9u; }
  }
  int s = 0;
  for (int j = 0; j < 8; ++j) s += acc[j];
  if (s == 0x7fffffff) out[0] = s;
}

// ---------------------------------------------------------------- tcgen05
__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ uint64_t desc_noswz(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFF) >> 4);
  d |= (uint64_t)((lbo & 0x3FFFF) >> 4) << 16;
  d |= (uint64_t)((sbo & 0x3FFFF) >> 4) << 32;
  d |= (uint64_t)1 << 46;  // descriptor version for tcgen05
  return d;                // layout type 0: no swizzle
}

template <int KIND>
__device__ __forceinline__ void mma_issue(uint32_t tmem, uint64_t ad, uint64_t bd, uint32_t idesc, uint32_t acc) {
  if (KIND == 0) {
    asm volatile("{\n.reg .pred p;\nsetp.ne.b32 p, %4, 0;\n"
                 "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n}\n"
                 :: "r"(tmem), "l"(ad), "l"(bd), "r"(idesc), "r"(acc));
  } else if (KIND == 1) {
    asm volatile("{\n.reg .pred p;\nsetp.ne.b32 p, %4, 0;\n"
                 "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n"
                 :: "r"(tmem), "l"(ad), "l"(bd), "r"(idesc), "r"(acc));
  }
#ifdef PROBE_I8
  else if (KIND == 2) {
    asm volatile("{\n.reg .pred p;\nsetp.ne.b32 p, %4, 0;\n"
                 "tcgen05.mma.cta_group::1.kind::i8 [%0], %1, %2, %3, p;\n}\n"
                 :: "r"(tmem), "l"(ad), "l"(bd), "r"(idesc), "r"(acc));
  }
#endif
}

// One CTA per SM. A = 128x32 bytes, B = 256x32 bytes (8-bit K-major, or 128x16/256x16 16-bit).
// All bytes equal, so the result does not depend on the core-matrix layout.
template <int KIND>
__global__ void __launch_bounds__(128, 1) k_tc(int iters, uint8_t abyte, uint8_t bbyte, uint16_t ahalf, uint16_t bhalf,
                                              uint32_t idesc, float* out_f, int* out_i, int* status) {
  __shared__ __align__(1024) uint8_t sA[128 * 32];
  __shared__ __align__(1024) uint8_t sB[256 * 32];
  __shared__ __align__(8) uint64_t mbar;
  __shared__ uint32_t tmem_slot;
  int tid = threadIdx.x, warp = tid >> 5;
  if (KIND == 1) {
    for (int i = tid; i < 128 * 16; i += 128) ((uint16_t*)sA)[i] = ahalf;
    for (int i = tid; i < 256 * 16; i += 128) ((uint16_t*)sB)[i] = bhalf;
  } else {
    for (int i = tid; i < 128 * 32; i += 128) sA[i] = abyte;
    for (int i = tid; i < 256 * 32; i += 128) sB[i] = bbyte;
  }
  if (tid == 0) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" :: "r"(smem_u32(&mbar)));
    asm volatile("fence.mbarrier_init.release.cluster;");
  }
  asm volatile("fence.proxy.async.shared::cta;");
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 256;" :: "r"(smem_u32(&tmem_slot)));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  asm volatile("tcgen05.fence::before_thread_sync;");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;");
  uint32_t tmem = tmem_slot;
  if (tid == 0) {
    uint64_t ad = desc_noswz(smem_u32(sA), 128, 256);
    uint64_t bd = desc_noswz(smem_u32(sB), 128, 256);
    for (int i = 0; i < iters; ++i) mma_issue<KIND>(tmem, ad, bd, idesc, i > 0 ? 1u : 0u);
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" :: "r"(smem_u32(&mbar)));
  }
  // bounded wait on the commit barrier (phase 0)
  uint32_t done = 0;
  uint64_t t0; asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t0));
  for (long it = 0; !done; ++it) {
    uint64_t t1; asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t1));
    if (t1 - t0 > 2000000000ull) break;
    asm volatile("{\n.reg .pred p;\nmbarrier.try_wait.parity.shared::cta.b64 p, [%1], 0;\nselp.u32 %0, 1, 0, p;\n}\n"
                 : "=r"(done) : "r"(smem_u32(&mbar)));
  }
  if (!done) atomicExch(status, 1);
  asm volatile("tcgen05.fence::after_thread_sync;");
  uint32_t v0, v1;
  uint32_t taddr = tmem + ((uint32_t)(warp * 32) << 16);
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x2.b32 {%0,%1}, [%2];" : "=r"(v0), "=r"(v1) : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;");
  if (blockIdx.x == 0) {
    if (KIND == 2) { out_i[tid * 2] = (int)v0; out_i[tid * 2 + 1] = (int)v1; }
    else { out_f[tid * 2] = __uint_as_float(v0); out_f[tid * 2 + 1] = __uint_as_float(v1); }
  }
  asm volatile("tcgen05.fence::before_thread_sync;");
  __syncthreads();
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 256;" :: "r"(tmem));
}

static uint32_t idesc_make(int cfmt, int afmt, int bfmt, int M, int N) {
  return ((uint32_t)cfmt << 4) | ((uint32_t)afmt << 7) | ((uint32_t)bfmt << 10) | ((uint32_t)(N >> 3) << 17) |
         ((uint32_t)(M >> 4) << 24);
}

template <typename F>
static float time_ms(F f) {
  cudaEvent_t a, b; cudaEventCreate(&a); cudaEventCreate(&b);
  f();  // warm
  cudaDeviceSynchronize();
  cudaEventRecord(a); f(); cudaEventRecord(b); cudaEventSynchronize(b);
  float ms; cudaEventElapsedTime(&ms, a, b);
  cudaEventDestroy(a); cudaEventDestroy(b);
  return ms;
}

int main() {
  cudaDeviceProp p; CK(cudaGetDeviceProperties(&p, 0));
  int clk = 0; cudaDeviceGetAttribute(&clk, cudaDevAttrClockRate, 0);
  printf("device %s sm_%d%d SMs %d L2 %d MB smem/block optin %zu clock %d kHz\n", p.name, p.major, p.minor,
         p.multiProcessorCount, p.l2CacheSize >> 20, p.sharedMemPerBlockOptin, clk);
  int nsm = p.multiProcessorCount;
  int *d_out, *d_i, *d_st; float* d_f;
  CK(cudaMalloc(&d_out, 64)); CK(cudaMalloc(&d_i, 4096)); CK(cudaMalloc(&d_f, 4096)); CK(cudaMalloc(&d_st, 4));
  CK(cudaMemset(d_st, 0, 4));
  const int blocks = nsm * 4, threads = 256, it = 4096;
  double warps = (double)blocks * threads / 32;
  {
    float ms = time_ms([&] { k_b1<<<blocks, threads>>>(it, d_out); });
    CK(cudaGetLastError());
    double ops = warps * it * 8 * 2.0 * 16 * 8 * 256;
    printf("mma.sync b1 and.popc m16n8k256: %.3f ms  %.1f TOPS (1-bit ops)\n", ms, ops / ms / 1e9);
  }
  {
    float ms = time_ms([&] { k_b1x<<<blocks, threads>>>(it, d_out); });
    CK(cudaGetLastError());
    double ops = warps * it * 8 * 2.0 * 16 * 8 * 256;
    printf("mma.sync b1 xor.popc m16n8k256: %.3f ms  %.1f TOPS (1-bit ops)\n", ms, ops / ms / 1e9);
  }
  {
    float ms = time_ms([&] { k_s8<<<blocks, threads>>>(it, d_out); });
    CK(cudaGetLastError());
    double ops = warps * it * 8 * 2.0 * 16 * 8 * 32;
    printf("mma.sync s8 m16n8k32: %.3f ms  %.1f TOPS\n", ms, ops / ms / 1e9);
  }
  {
    float ms = time_ms([&] { k_e4m3<<<blocks, threads>>>(it, d_out); });
    CK(cudaGetLastError());
    double ops = warps * it * 8 * 2.0 * 16 * 8 * 32;
    printf("mma.sync e4m3 m16n8k32: %.3f ms  %.1f TFLOPS\n", ms, ops / ms / 1e9);
  }
  {
    float ms = time_ms([&] { k_popc<<<blocks, threads>>>(it * 4, d_out); });
    CK(cudaGetLastError());
    double ops = (double)blocks * threads * it * 4 * 8 * 2.0 * 32;
    printf("CUDA-core xor+popc: %.3f ms  %.1f TOPS (1-bit ops)\n", ms, ops / ms / 1e9);
  }
  // tcgen05: M=128 N=256 K=32 (8-bit) / K=16 (16-bit)
  const int tcit = 8192;
  {
    uint32_t id = idesc_make(1, 0, 0, 128, 256);
    float ms = time_ms([&] { k_tc<0><<<nsm, 128>>>(tcit, 0x38, 0x38, 0, 0, id, d_f, d_i, d_st); });
    CK(cudaGetLastError());
    double ops = (double)nsm * tcit * 2.0 * 128 * 256 * 32;
    printf("tcgen05 f8f6f4 e4m3 128x256x32: %.3f ms  %.1f TFLOPS\n", ms, ops / ms / 1e9);
  }
  {
    uint32_t id = idesc_make(1, 1, 1, 128, 256);
    float ms = time_ms([&] { k_tc<1><<<nsm, 128>>>(tcit, 0, 0, 0x3F80, 0x3F80, id, d_f, d_i, d_st); });
    CK(cudaGetLastError());
    double ops = (double)nsm * tcit * 2.0 * 128 * 256 * 16;
    printf("tcgen05 f16 bf16 128x256x16: %.3f ms  %.1f TFLOPS\n", ms, ops / ms / 1e9);
  }
#ifdef PROBE_I8
  {
    uint32_t id = idesc_make(2, 1, 1, 128, 256);
    float ms = time_ms([&] { k_tc<2><<<nsm, 128>>>(tcit, 1, 1, 0, 0, id, d_f, d_i, d_st); });
    CK(cudaGetLastError());
    double ops = (double)nsm * tcit * 2.0 * 128 * 256 * 32;
    printf("tcgen05 i8 128x256x32: %.3f ms  %.1f TOPS\n", ms, ops / ms / 1e9);
  }
#endif
  // exactness: e4m3 15 x 1 summed 32 per instruction; n instructions -> 480 n exactly if fp32 accumulate is exact
  for (int n : {1, 100, 4096, 20000, 34952}) {
    uint32_t id = idesc_make(1, 0, 0, 128, 256);
    k_tc<0><<<1, 128>>>(n, 0x57, 0x38, 0, 0, id, d_f, d_i, d_st);
    CK(cudaDeviceSynchronize());
    float h[256]; CK(cudaMemcpy(h, d_f, sizeof(h), cudaMemcpyDeviceToHost));
    int bad = 0; for (int i = 0; i < 256; ++i) if (h[i] != 480.0f * n) ++bad;
    printf("exact e4m3 15*1 n=%d: expect %.0f got %.1f bad=%d\n", n, 480.0 * n, h[0], bad);
  }
  // mixed-sign: A=15, B=-1 after positive accumulation? use bf16 255 * 1 over 16 -> 4080 per instr
  for (int n : {1, 1000, 4112}) {
    uint32_t id = idesc_make(1, 1, 1, 128, 256);
    k_tc<1><<<1, 128>>>(n, 0, 0, 0x437F /*255*/, 0x3F80, id, d_f, d_i, d_st);
    CK(cudaDeviceSynchronize());
    float h[256]; CK(cudaMemcpy(h, d_f, sizeof(h), cudaMemcpyDeviceToHost));
    int bad = 0; for (int i = 0; i < 256; ++i) if (h[i] != 4080.0f * n) ++bad;
    printf("exact bf16 255*1 n=%d: expect %.0f got %.1f bad=%d\n", n, 4080.0 * n, h[0], bad);
  }
  int st; CK(cudaMemcpy(&st, d_st, 4, cudaMemcpyDeviceToHost));
  printf("status %d\n", st);
  return 0;
}
