// Internal launchers of the integer GEMM kernels.
#pragma once
#include "common.cuh"

namespace fqt1 {

// tcgen05 path (gemm_tc.cu)
struct TcArgs;
cudaError_t launch_fwd_tc(const uint32_t* A, const uint32_t* B, int64_t M, int64_t D, int64_t K, const float* gamma,
                          const float* bias, int32_t* acc, float* y, int32_t* status, cudaStream_t s);
// Implicit-GEMM forward of a stride-1 "same" convolution from pixel-major sign words xp
// [N][H][W][C / 32] and tap-major weight signs wt [D][words(k k C)] (k' = t C + c); the shapes
// implicit_conv_supported accepts.
bool implicit_conv_supported(int64_t N, int64_t C, int64_t H, int64_t W, int64_t kh, int64_t kw, int64_t stride,
                             int64_t pad);
cudaError_t launch_fwd_implicit_tc(const uint32_t* xp, const uint32_t* wt, int N, int C, int H, int W, int k, int pad,
                                   int64_t D, const float* gamma, const float* bias, int32_t* acc, float* y,
                                   int32_t* status, cudaStream_t s);
cudaError_t launch_codes_tc_simple(int bits, const uint8_t* Q, int64_t ldq, int64_t max_rows, const int32_t* count,
                                   int64_t rows_per_count, const uint32_t* Sg, int64_t n_s, int64_t L, int epi,
                                   int splits, int32_t* acc, float* out, int64_t ldo, const int32_t* kept_idx,
                                   const float* scale, const float* zero, const int32_t* cs, int64_t rpg,
                                   int32_t* status, cudaStream_t s, const uint8_t* Be = nullptr,
                                   int64_t ldbe = 0);
enum : int { GEMM_EPI_ACC32 = 1, GEMM_EPI_RED = 2, GEMM_EPI_DX = 3 };
// The same product with EPI_ACC32 accumulators column-major: acc[n * ld + r] (ld >= max_rows),
// each warp's 32 rows of a column stored as one line straight from the TMEM registers; acc_bits
// 32 (int32) or 16 (int16, when every sum fits).  Be (optional): e4m3 sign(W)^T rows [n_s][ldbe]
// bytes by TMA instead of the packed columns Sg.
cudaError_t launch_codes_tc_colmajor(int bits, const uint8_t* Q, int64_t ldq, int64_t max_rows, const int32_t* count,
                                     int64_t rows_per_count, const uint32_t* Sg, int64_t n_s, int64_t L,
                                     void* acc, int acc_bits, int64_t ld, int32_t* status, cudaStream_t s,
                                     const uint8_t* Be = nullptr, int64_t ldbe = 0);
// Bte: e4m3 sign(W)^T rows [K][ldbte] bytes, or null for the packed sign(W) columns Sg.
// nhwc: dx in memory order N, H, W, C.
cudaError_t launch_fold_tc(int bits, const uint8_t* Q, int64_t ldq, int64_t max_rows, const int32_t* count,
                           const uint32_t* Sg, int64_t K, int64_t D, const int32_t* kept_idx, const float* scale,
                           const float* zero, const int32_t* cs, const int32_t* slot_of_group, float* dx, int N, int C,
                           int H, int W, int kh, int kw, int stride, int pad, int Ho, int Wo, int32_t* status,
                           cudaStream_t s, const uint8_t* Bte = nullptr, int64_t ldbte = 0, int nhwc = 0);
// fqt1_fwd_gemm's kernel with the first operand stage's arrive withheld: its bounded waits
// (20 ms) expire, FQT1_DEV_TIMEOUT is set in *status and the kernel returns normally.
cudaError_t launch_fwd_lost_arrive_tc(const uint32_t* A, const uint32_t* B, int64_t M, int64_t D, int64_t K,
                                      const float* gamma, float* y, int32_t* status, cudaStream_t s);
// Forward with B = e4m3 sign(W) rows [D][ldbe] bytes (+1 = 0x38, -1 = 0xB8, bytes past K zero).
cudaError_t launch_fwd_e4m3w_tc(const uint32_t* A, const uint8_t* Be, int64_t ldbe, int64_t M, int64_t D, int64_t K,
                                const float* gamma, const float* bias, int32_t* acc, float* y, int32_t* status,
                                cudaStream_t s);
// Bytes of the fused Folder's tables (tap offsets, folded colsums, per-sample constants); the
// fused path needs this to be at most 36864.
inline int64_t fold_table_bytes(int64_t H, int64_t W, int64_t kh, int64_t kw, int64_t Ho, int64_t Wo) {
  const int64_t khw = kh * kw, cb = 128 / khw;
  return 4 * (H * W * khw + cb * H * W + cb * khw) + 12 * (128 / (Ho * Wo));
}
// grad_weight with the split-K reduction and the dequantization in the kernel: the splits of
// an output tile form a thread-block cluster of `splits` (<= 8) CTAs that add their partial
// tiles through distributed shared memory.  acc [capacity][K] receives the int32 sums (rows past
// the kept count 0), dw [D][K] the dequantized rows (pruned channels 0).  Be (optional): the
// signs of X_u^T as e4m3 bytes [K][ldbe] (by TMA into the operand ring) instead of Sx.
cudaError_t launch_wgrad_cluster_tc(int bits, const uint8_t* Q, int64_t ldq, int64_t capacity, const int32_t* count,
                                    const uint32_t* Sx, int64_t K, int64_t M, int splits, int32_t* acc, float* dw,
                                    int64_t D, const int32_t* kept_idx, const int32_t* slot_of_group,
                                    const float* scale, const float* zero, const int32_t* cs, int32_t* status,
                                    cudaStream_t s, const uint8_t* Be = nullptr, int64_t ldbe = 0);
// Forward with A = e4m3 sign(X_u) rows [M][ldxe] and B = e4m3 sign(W) rows [D][ldbe] bytes
// (+1 = 0x38, -1 = 0xB8, bytes past K zero), both straight from TMA.
cudaError_t launch_fwd_e4m3x_tc(const uint8_t* Xe, int64_t ldxe, const uint8_t* Be, int64_t ldbe, int64_t M, int64_t D,
                                int64_t K, const float* gamma, const float* bias, int32_t* acc, float* y,
                                int32_t* status, cudaStream_t s);
// Cluster size for launch_wgrad_cluster_tc: the largest (<= 8, <= k_tiles) whose out_tiles
// clusters fit on the GPU at once.
int wgrad_cluster_size(int bits, int64_t out_tiles, int64_t k_tiles);
// Contraction elements per pipeline stage of the code x sign products (the grad_input and
// grad_weight GEMMs): split counts and the exactness bound are counted in these stages.
constexpr int kCodesStageK = 256;
// Largest contraction one CTA may sum in fp32 and stay exact: partial sums below 2^24.
inline int64_t exact_chunk(int bits) { return (int64_t)((1 << 24) / ((1 << bits) - 1)); }

}  // namespace fqt1
