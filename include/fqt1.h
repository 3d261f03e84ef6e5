/*
 * libfqt1 -- one fully quantized 1-bit training step of a linear or
 * convolution layer on an sm_103a GPU (1-Bit FQT, arXiv 2408.14267).
 *
 * Conventions for every entry point
 * ---------------------------------
 *  - Pointers are DEVICE pointers unless stated otherwise.  The caller owns and
 *    allocates every buffer; the library allocates nothing, never
 *    synchronizes, and enqueues all work on `stream` (a cudaStream_t, NULL
 *    for the legacy default stream).
 *  - Return value: host-side validation / launch status.  On any error no
 *    kernel has been launched for that call.
 *  - Conditions found on the device (non-finite gradient values, an expired
 *    wait) are OR-ed into `*dev_status` (int32, zeroed by the caller); read it
 *    after synchronizing.
 *  - Sizes are element counts; every float / int buffer must be 16-byte
 *    aligned and rows described by an `ld` must keep that alignment.
 *
 * Data layouts
 * ------------
 *  Packed signs ("bits"): a [rows, cols] sign matrix is stored as uint32 words
 *  [rows][fqt1_packed_words(cols)]; bit e % 32 of word e / 32 is 1 iff
 *  x > 0 (sign +1, Sec. 5.1), least significant bit first.  Padding bits and
 *  padding words are 0.  "row bits" pack a matrix along its columns, "col
 *  bits" pack its transpose (one packed row per column).
 *  Gradient codes: uint8 integers q in [0, 2^b - 1] (Sec. 3.2), rows of
 *  `ld_codes` bytes.  PSQ codes are [capacity * rows_per_group][ld >= D] in
 *  kept order; PCQ codes are [capacity][ld >= M] (one row per kept channel,
 *  samples contiguous).
 *  Convolutions use the Unfolder of App. C: row m = (n*Ho + oh)*Wo + ow,
 *  column k = (c*kh + i)*kw + j; the layer output / gradient y, gy are
 *  [N*Ho*Wo, D] (NHWC rows).
 */
#ifndef FQT1_H
#define FQT1_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  FQT1_OK = 0,
  FQT1_ERR_INVALID_ARG = 1,  /* null pointer, bad size, bad bits/mode        */
  FQT1_ERR_MISALIGNED = 2,   /* a pointer or ld breaks 16-byte alignment      */
  FQT1_ERR_UNSUPPORTED = 3,  /* valid but outside the implemented range       */
  FQT1_ERR_WORKSPACE = 4,    /* workspace missing or too small                */
  FQT1_ERR_CUDA = 5          /* a CUDA runtime call failed (see fqt1_last_cuda_error) */
} fqt1_status;

/* Bits OR-ed into *dev_status by kernels. */
#define FQT1_DEV_NONFINITE 0x100 /* a gradient value was NaN or +-Inf          */
#define FQT1_DEV_TIMEOUT 0x200   /* a bounded wait expired; results invalid    */

/* How AGP draws its masks m_i (Sec. 5.2) from the keep probabilities p_i. */
typedef enum {
  FQT1_SEL_SYSTEMATIC = 0, /* one uniform offset; P(keep i) = p^_i exactly, kept count
                              floor or ceil of sum p^ (default)                        */
  FQT1_SEL_BERNOULLI = 1,  /* independent m_i ~ Bern(p^_i)                             */
  FQT1_SEL_TOPK = 2        /* the floor(n/b) largest ranges, p^ = 1 (App. B, biased)   */
} fqt1_select;

/* AGP settings of one gradient branch. */
typedef struct {
  int32_t bits;            /* b in {1, 2, 4, 8}: bits of a kept group; keep ratio 1/b   */
  int32_t mode;            /* fqt1_select                                               */
  uint64_t seed;           /* key of the counter-based generator (Philox4x32-10)        */
  int64_t rows_per_group;  /* PSQ only: rows of one sample group (1 for linear layers,
                              Ho*Wo for convolutions); must divide M                    */
} fqt1_agp_params;

/* One quantized gradient branch (PSQ or PCQ); every array is caller-owned.
 * n = number of groups (M / rows_per_group for PSQ, D for PCQ);
 * capacity = fqt1_kept_capacity(n, bits, mode). */
typedef struct {
  float* group_min;        /* [n]  Z_i = min of the group (Sec. 3.2)                  */
  float* group_range;      /* [n]  R_i = max - min                                    */
  double* p_hat;           /* [n]  keep probability actually used, P_i / 2^32         */
  int32_t* slot_of_group;  /* [n]  position of group i in the kept list, -1 if pruned  */
  int32_t* kept_idx;       /* [capacity] kept group ids, ascending; -1 past the count  */
  int32_t* kept_count;     /* [1]  number of kept groups                               */
  float* scale;            /* [capacity] S' = R / (B p^) of each kept group            */
  float* zero;             /* [capacity] Z' = Z / p^ of each kept group                */
  uint8_t* codes;          /* codes of the kept groups (layout above)                  */
  int64_t ld_codes;        /* bytes between code rows, multiple of 16                  */
} fqt1_qgrad;

/* ---------------------------------------------------------------- helpers */
/* uint32 words of one packed row of n signs: ceil(n/32) rounded up to a multiple of 4. */
int64_t fqt1_packed_words(int64_t n);
/* Upper bound of kept groups: n for b = 1 or BERNOULLI, else ceil(n / b). */
int64_t fqt1_kept_capacity(int64_t n, int32_t bits, int32_t mode);
/* Smallest legal ld_codes for rows of n codes (n rounded up to 16). */
int64_t fqt1_codes_ld(int64_t n);
/* Workspace bytes for fqt1_scq_quantize / fqt1_agp_quantize_grad (which = 0) and
 * fqt1_bwd_weight_gemm (which = 1) on an [M, D] gradient / [D, K] weight. */
size_t fqt1_workspace_size(int32_t which, int64_t M, int64_t D, int64_t K, int32_t rows_per_group);
/* Text of the last CUDA error seen by the calling host thread. */
const char* fqt1_last_cuda_error(void);
/* Number of kernels this library has enqueued since it was loaded (all threads). */
int64_t fqt1_kernel_launches(void);

/* ------------------------------------------------------------ forward side */
/* Binarize and pack (Sec. 5.1; row / column encoders of App. C, Algorithm 2).
 * x: [rows, cols] fp32 with leading dimension ld >= cols.
 * row_bits: [rows][fqt1_packed_words(cols)] or NULL.
 * col_bits: [cols][fqt1_packed_words(rows)] or NULL.
 * colsum:   [cols] int32, colsum[c] = sum_r sign(x[r, c]), or NULL.
 * At least one output must be given.  For the weight W [D, K] the three
 * outputs feed the forward GEMM, grad_input GEMM and its dequantization; for
 * a linear input X [M, K] they feed the forward GEMM, grad_weight GEMM and its
 * dequantization. */
fqt1_status fqt1_binarize_pack(const float* x, int64_t rows, int64_t cols, int64_t ld, uint32_t* row_bits,
                               uint32_t* col_bits, int32_t* colsum, void* stream);

/* Unfolder of App. C fused with sign and pack: x [N, C, H, W] fp32 ->
 * the packed signs of X_u [M = N*Ho*Wo, K = C*kh*kw]; positions in the zero
 * padding count as x = 0, i.e. sign -1.  Outputs as in fqt1_binarize_pack
 * for the matrix X_u (row_bits [M][words(K)], col_bits [K][words(M)],
 * colsum [K] over all M rows). */
fqt1_status fqt1_im2col(const float* x, int32_t N, int32_t C, int32_t H, int32_t W, int32_t kh, int32_t kw,
                        int32_t stride, int32_t pad, uint32_t* row_bits, uint32_t* col_bits, int32_t* colsum,
                        void* stream);

/* Implicit-GEMM convolution forward (the Unfolder of App. C left implicit).
 * The binary product of a stride-1 "same" convolution (kh = kw = 2 pad + 1) is
 * computed without materializing X_u: the contraction runs over kernel taps
 * and channels, k' = t C + c for tap t = i kw + j.  Each A tile is read from
 * pixel-major sign words, shifted by the tap, and taps in the zero padding read
 * sign -1 (as in fqt1_im2col).  The integer result equals fqt1_fwd_gemm on the
 * unfolded matrix, since it is the same sum in another order.
 *
 * fqt1_pack_pixels: x [N, C, H, W] fp32 -> x_pix [N*H*W][fqt1_packed_words(C)];
 *   word b of pixel p = (n H + h) W + w has bit e set iff x[n, 32 b + e, h, w] > 0.
 *   C must be a multiple of 128 (FQT1_ERR_UNSUPPORTED otherwise); x_pix 16-byte
 *   aligned.
 * fqt1_pack_weight_taps: w [D, C, kh, kw] fp32 -> w_taps
 *   [D][fqt1_packed_words(kh*kw*C)]; bit e of word t C / 32 + b of row d is set
 *   iff w[d, 32 b + e, i, j] > 0 (t = i kw + j); padding words are 0.  C must be
 *   a multiple of 32.
 * fqt1_conv_implicit_supported: 1 if fqt1_conv_fwd_implicit accepts the shape:
 *   stride 1, kh = kw = 2 pad + 1, C a multiple of 128, kh kw C < 2^24, and the
 *   output pixels tile by 128 rows as whole images (H W divides 128) or as whole
 *   image rows (W divides 128 and 128 / W divides H).  Otherwise 0.
 * fqt1_conv_fwd_implicit: acc[m, d] = sum_k sign(X_u)[m, k] sign(W)[d, k] for
 *   output pixel m = (n H + h) W + w; y = gamma[d] acc (+ bias[d]) as in
 *   fqt1_fwd_gemm_bias.  acc may be NULL; gamma and y are required.
 *   FQT1_ERR_UNSUPPORTED for a shape that fqt1_conv_implicit_supported rejects.
 * Buffers are caller-owned device memory and all three calls are asynchronous
 * on `stream`. */
fqt1_status fqt1_pack_pixels(const float* x, int32_t N, int32_t C, int32_t H, int32_t W, uint32_t* x_pix,
                             void* stream);
fqt1_status fqt1_pack_weight_taps(const float* w, int64_t D, int32_t C, int32_t kh, int32_t kw, uint32_t* w_taps,
                                  void* stream);
int32_t fqt1_conv_implicit_supported(int32_t N, int32_t C, int32_t H, int32_t W, int32_t kh, int32_t kw,
                                     int32_t stride, int32_t pad);
fqt1_status fqt1_conv_fwd_implicit(const uint32_t* x_pix, const uint32_t* w_taps, int32_t N, int32_t C, int32_t H,
                                   int32_t W, int32_t kh, int32_t kw, int32_t stride, int32_t pad, int64_t D,
                                   const float* gamma, const float* bias, int32_t* acc, float* y, void* stream);

/* Sign planes of a contiguous x (App. C Unfolder, in two passes).
 * fqt1_pack_planes: x [N, C, H, W] fp32 (contiguous, 16-byte aligned) -> planes
 *   [N][C][ceil(H W / 32)] words: bit e of word q of plane (n, c) is set iff
 *   x[n, c, pixel 32 q + e] > 0 (pixel = h W + w), bits past H W clear; the
 *   layout fqt1_pack_planes_nhwc writes and fqt1_im2col_planes reads.  One
 *   streaming pass over x.
 * fqt1_im2col_path: how fqt1_im2col serves the shape.  2: tiles of whole images
 *   (stride-1 "same" convolutions whose H W divides 128 or is 256), one pass over
 *   x.  1: tiles of up to 128 output pixels, each reading its input region; then
 *   fqt1_pack_planes followed by fqt1_im2col_planes gives the same outputs from
 *   32 times fewer bytes.  3: a pointwise convolution (1 x 1 window, no padding):
 *   one pass over x, which fqt1_im2col reads directly (fqt1_im2col_planes serves
 *   it with region tiles).  0: a per-element gather (regions too large; x must be
 *   given).  -1: a shape fqt1_im2col rejects (invalid, or N C H W, N Ho Wo or
 *   H + 2 pad reaching 2^31). */
fqt1_status fqt1_pack_planes(const float* x, int32_t N, int32_t C, int32_t H, int32_t W, uint32_t* planes,
                             void* stream);
int32_t fqt1_im2col_path(int32_t N, int32_t C, int32_t H, int32_t W, int32_t kh, int32_t kw, int32_t stride,
                         int32_t pad);

/* Channels-last inputs (no counterpart in the paper; the layout of x only).
 * fqt1_pack_planes_nhwc: x with memory order N, H, W, C (a channels-last
 *   [N, C, H, W] tensor), C a multiple of 32 -> planes [N][C][ceil(H W / 32)]
 *   words: bit e of word q of plane (n, c) is set iff x[n, c, pixel 32 q + e] > 0
 *   (pixel = h W + w), bits past H W clear.  x 16-byte aligned.
 * fqt1_im2col_planes: fqt1_im2col from those plane bits instead of x, same
 *   outputs bit for bit.  FQT1_ERR_UNSUPPORTED for shapes whose tiles read
 *   more input than fits in shared memory (fqt1_im2col then reads x itself). */
fqt1_status fqt1_pack_planes_nhwc(const float* x, int32_t N, int32_t C, int32_t H, int32_t W, uint32_t* planes,
                                  void* stream);
fqt1_status fqt1_im2col_planes(const uint32_t* planes, int32_t N, int32_t C, int32_t H, int32_t W, int32_t kh,
                               int32_t kw, int32_t stride, int32_t pad, uint32_t* row_bits, uint32_t* col_bits,
                               int32_t* colsum, void* stream);
/* fqt1_col2im and fqt1_bwd_input_fold with dx in channels-last memory order
 * (N, H, W, C): the same values, element (n, c, h, w) at ((n H + h) W + w) C + c.
 * fqt1_col2im_nhwc returns FQT1_ERR_UNSUPPORTED for shapes that fqt1_col2im
 * serves with its untiled kernel. */
fqt1_status fqt1_col2im_nhwc(const int32_t* acc, const fqt1_qgrad* psq, const int32_t* colsum_w, int32_t N,
                             int32_t C, int32_t H, int32_t W, int32_t kh, int32_t kw, int32_t stride, int32_t pad,
                             float* dx, void* stream);
fqt1_status fqt1_bwd_input_fold_nhwc(const fqt1_qgrad* psq, const uint32_t* sw_col, const int32_t* colsum_w,
                                     int32_t N, int32_t C, int32_t H, int32_t W, int32_t kh, int32_t kw,
                                     int32_t stride, int32_t pad, int64_t D, const fqt1_agp_params* p, float* dx,
                                     void* stream);

/* Binarized forward GEMM (Sec. 5.1, App. C "binary multiplication"):
 * acc[m, j] = sum_k sign(X)[m, k] sign(W)[j, k], y[m, j] = gamma[j] * acc[m, j] (fp32).
 * sx_row: [M][words(K)], sw_row: [D][words(K)], gamma: [D].
 * acc: [M][D] int32 or NULL; y: [M][D] fp32 (row stride D) or NULL, at least one of
 * the two given (gamma may be NULL when y is). */
fqt1_status fqt1_fwd_gemm(const uint32_t* sx_row, const uint32_t* sw_row, int64_t M, int64_t D, int64_t K,
                          const float* gamma, int32_t* acc, float* y, void* stream);

/* Test of the failure path (no counterpart in the paper): the kernel of fqt1_fwd_gemm
 * with every bounded wait cut to 20 ms and the arrive that hands its first operand stage to
 * the tensor cores withheld, so the wait for it runs out.  The kernel then sets
 * FQT1_DEV_TIMEOUT in *dev_status (int32, zeroed by the caller), waits for its in-flight copies,
 * frees its tensor memory and returns; the context stays usable.  y receives unspecified
 * values.  Arguments as fqt1_fwd_gemm (gamma and y required, no acc).  Meant for tests that
 * check that a caller sees an expired wait as a status, not as a hang. */
fqt1_status fqt1_test_expired_wait(const uint32_t* sx_row, const uint32_t* sw_row, int64_t M, int64_t D, int64_t K,
                                   const float* gamma, float* y, int32_t* dev_status, void* stream);

/* fqt1_fwd_gemm with a per-channel bias: y[m, j] = gamma[j] * acc[m, j] + bias[j]
 * (fp32 multiply, then fp32 add).  The paper's layer (Sec. 5.1) has the scale
 * Gamma only; the bias is the usual extension of a linear or convolution layer
 * (Algorithm 1 omits it).  bias: [D] fp32, 16-byte aligned, or NULL (then the
 * call equals fqt1_fwd_gemm); a bias needs y. */
fqt1_status fqt1_fwd_gemm_bias(const uint32_t* sx_row, const uint32_t* sw_row, int64_t M, int64_t D, int64_t K,
                               const float* gamma, const float* bias, int32_t* acc, float* y, void* stream);

/* e4m3 copies of sign(W) for the products' B operand (no counterpart in the
 * paper: the same +-1 values in the tensor cores' byte format, so that the
 * products load B with TMA instead of expanding packed bits in every CTA).
 * fqt1_expand_signs_e4m3: packed signs bits [rows][fqt1_packed_words(n)] (as
 *   written by fqt1_binarize_pack) -> out [rows][ld_out] bytes: 0x38 (+1) where
 *   the bit is set, 0xB8 (-1) where it is clear, 0 for columns n .. ld_out - 1.
 *   ld_out >= n and a multiple of 16; both pointers 16-byte aligned.
 * fqt1_fwd_gemm_e4m3w: fqt1_fwd_gemm_bias with sign(W) given as w_e4m3
 *   [D][ld_w] (the row packing expanded); gamma and y required, acc and bias
 *   may be NULL.  Results equal fqt1_fwd_gemm_bias bit for bit.
 * fqt1_bwd_input_fold_e4m3w: fqt1_bwd_input_fold with sign(W)^T given as
 *   wt_e4m3 [K][ld_wt] (the column packing expanded, ld_wt >= D).  Results
 *   equal fqt1_bwd_input_fold bit for bit. */
fqt1_status fqt1_expand_signs_e4m3(const uint32_t* bits, int64_t rows, int64_t n, uint8_t* out, int64_t ld_out,
                                   void* stream);
/* fqt1_binarize_pack with the e4m3 bytes of the signs as two more optional
 * outputs, written by the same pass over x where its rows are a multiple of 4
 * floats (otherwise the packed outputs, which must then be given, are expanded
 * by fqt1_expand_signs_e4m3): row_e4m3 [rows][ld_re] (ld_re >= cols, columns
 * past cols 0) and col_e4m3 [cols][ld_ce] (ld_ce >= rows, rows past `rows` 0);
 * ld_re and ld_ce multiples of 16, all pointers 16-byte aligned. */
fqt1_status fqt1_binarize_pack_e4m3(const float* x, int64_t rows, int64_t cols, int64_t ld, uint32_t* row_bits,
                                    uint32_t* col_bits, int32_t* colsum, uint8_t* row_e4m3, int64_t ld_re,
                                    uint8_t* col_e4m3, int64_t ld_ce, void* stream);
fqt1_status fqt1_fwd_gemm_e4m3w(const uint32_t* sx_row, const uint8_t* w_e4m3, int64_t ld_w, int64_t M, int64_t D,
                                int64_t K, const float* gamma, const float* bias, int32_t* acc, float* y,
                                void* stream);
fqt1_status fqt1_bwd_input_fold_e4m3w(const fqt1_qgrad* psq, const uint8_t* wt_e4m3, int64_t ld_wt,
                                      const int32_t* colsum_w, int32_t N, int32_t C, int32_t H, int32_t W,
                                      int32_t kh, int32_t kw, int32_t stride, int32_t pad, int64_t D,
                                      const fqt1_agp_params* p, float* dx, void* stream);

/* e4m3 copies of sign(X_u) for the forward and grad_weight products (no
 * counterpart in the paper: the Unfolder's +-1 values of App. C in the tensor
 * cores' byte format, so that both products load their sign operand with TMA
 * and expand nothing; 8 times the bytes of the packed signs).
 * fqt1_im2col_e4m3: the Unfolder of fqt1_im2col writing x_row [M][ld_row]
 *   (row m = output pixel, byte k = column of X_u; ld_row >= K rounded up to 16)
 *   and x_col [K][ld_col] (the transpose; ld_col >= M rounded up to 16) instead
 *   of the packed words: 0x38 (+1), 0xB8 (-1), and 0 from the valid length to
 *   the next multiple of 16; colsum [K] as in fqt1_im2col.  Each output may be
 *   NULL (x_row or x_col must be given); pointers 16-byte aligned.  Serves the
 *   shapes for which fqt1_im2col_path returns 2; others give
 *   FQT1_ERR_UNSUPPORTED before any launch.
 * fqt1_fwd_gemm_e4m3x: the forward product of Sec. 5.1 with both operands as
 *   e4m3 signs: x_e4m3 [M][ld_x] (from fqt1_im2col_e4m3, or the row_e4m3 of
 *   fqt1_binarize_pack_e4m3 for a linear X) and w_e4m3 [D][ld_w]; bytes past K
 *   must be 0 in at least one of them.  gamma, bias, acc and y as in
 *   fqt1_fwd_gemm_bias; results equal it bit for bit.
 * fqt1_bwd_weight_gemm_e4m3x: fqt1_bwd_weight_gemm with sign(X_u)^T given as
 *   x_col_e4m3 [K][ld_xc] bytes (ld_xc >= M rounded up to 16); results equal it
 *   bit for bit. */
fqt1_status fqt1_im2col_e4m3(const float* x, int32_t N, int32_t C, int32_t H, int32_t W, int32_t kh, int32_t kw,
                             int32_t stride, int32_t pad, uint8_t* x_row, int64_t ld_row, uint8_t* x_col,
                             int64_t ld_col, int32_t* colsum, void* stream);
fqt1_status fqt1_fwd_gemm_e4m3x(const uint8_t* x_e4m3, int64_t ld_x, const uint8_t* w_e4m3, int64_t ld_w, int64_t M,
                                int64_t D, int64_t K, const float* gamma, const float* bias, int32_t* acc, float* y,
                                void* stream);
fqt1_status fqt1_bwd_weight_gemm_e4m3x(const fqt1_qgrad* pcq, const uint8_t* x_col_e4m3, int64_t ld_xc,
                                       const int32_t* colsum_x, int64_t M, int64_t D, int64_t K,
                                       const fqt1_agp_params* p, int32_t* acc, float* dw, void* stream);

/* ------------------------------------------------ layer parameters and STE */
/* Gradients of the layer's scale Gamma (Sec. 5.1: y = (sign(X) sign(W)^T) (.)
 * Gamma, Gamma learnable) and of its bias:
 *   dgamma[j] = sum_m gy[m, j] acc[m, j],   dbias[j] = sum_m gy[m, j].
 * gy: [M][D] fp32 (the gradient of y); acc: [M][D] int32, the forward
 * accumulators (fqt1_fwd_gemm's acc), needed for dgamma; dgamma, dbias: [D]
 * fp32, either may be NULL, overwritten.  The sums run in a fixed order (fp32
 * within 256-row chunks, fp64 over the chunks), so the results are reproducible.
 * ws: fqt1_scale_bias_workspace(M, D) bytes, 16-byte aligned, caller-owned. */
size_t fqt1_scale_bias_workspace(int64_t M, int64_t D);
fqt1_status fqt1_scale_bias_grad(const float* gy, const int32_t* acc, int64_t M, int64_t D, float* dgamma,
                                 float* dbias, void* ws, size_t ws_bytes, void* stream);

/* Clipped straight-through estimator of sign() (the STE cited in Sec. 3.1):
 * dx[i] = dx[i] if |x[i]| <= t else 0, in place, for i < n.  Without this call
 * the gradient passes sign() unchanged (the identity STE).  x, dx: [n] fp32,
 * 16-byte aligned; t >= 0 (NaN x gives 0). */
fqt1_status fqt1_ste_clip(const float* x, float* dx, int64_t n, float t, void* stream);

/* ----------------------------------------------------------- gradient side */
/* Prepare a workspace of fqt1_agp_quantize_grad / fqt1_scq_quantize: fill its
 * ws_bytes bytes with 0xFF on `stream` (the initial value of the range keys,
 * which both take atomicMin).  Needed once per buffer: every call that returns
 * FQT1_OK leaves the keys it used at 0xFF again (the selection kernel resets
 * each key after reading it), so one workspace serves any sequence of calls and
 * shapes that fit it.  Call it again after a call that failed once its kernels
 * had been launched (a launch error), as that may leave keys behind.
 * Errors: FQT1_ERR_INVALID_ARG for a null ws or ws_bytes 0; FQT1_ERR_CUDA if
 * the fill cannot be queued. */
fqt1_status fqt1_scq_workspace_init(void* ws, size_t ws_bytes, void* stream);

/* AGP on one grouping (Sec. 5.2): ranges of G = gy (.) gamma (gamma may be
 * NULL), keep probabilities, masks, and stochastic rounding of the kept
 * groups to `bits`-bit codes with scales S' and zero points Z'.
 * g: [M, D] fp32 row-major.  group_axis 0 = sample groups (PSQ: rounding takes
 * word m*D + j of generator stream 0, masks stream 2), 1 = channels (PCQ: word
 * j*M + m of stream 1, masks stream 3).
 * ws: fqt1_workspace_size(0, ...) bytes, initialised by fqt1_scq_workspace_init
 * (a workspace holding anything else gives wrong ranges). */
fqt1_status fqt1_agp_quantize_grad(const float* g, int64_t M, int64_t D, int32_t group_axis, const float* gamma,
                                   const fqt1_agp_params* p, fqt1_qgrad* out, void* ws, size_t ws_bytes,
                                   int32_t* dev_status, void* stream);

/* Sample-Channel joint Quantization (Sec. 5.3): both AGP branches of one
 * gradient from a single range pass and a single quantization pass:
 * psq groups rows (rows_per_group from p_sample), pcq groups columns. */
fqt1_status fqt1_scq_quantize(const float* g, int64_t M, int64_t D, const float* gamma,
                              const fqt1_agp_params* p_sample, const fqt1_agp_params* p_channel,
                              fqt1_qgrad* psq, fqt1_qgrad* pcq, void* ws, size_t ws_bytes, int32_t* dev_status,
                              void* stream);

/* Allocation-free fqt1_scq_quantize.  The paper has no counterpart: this only
 * changes where the scratch memory lives.  It is meant for callers that cannot
 * allocate device memory when they quantize (a plugin interface that only
 * passes in the tensors, or a memory pool frozen after warm-up), so they cannot
 * supply `ws`.  The range-pass scratch is instead a fixed array of
 * FQT1_NOALLOC_SCRATCH_KEYS uint32 (64 KiB) inside the library, held on every
 * device that loads it until the process exits.
 *  - Sizes: 2 * (M / rows_per_group) + 2 * D must not exceed
 *    FQT1_NOALLOC_SCRATCH_KEYS; larger calls return FQT1_ERR_UNSUPPORTED and
 *    fqt1_last_cuda_error() names the limit.
 *  - The first call on a device (the device current on the calling thread,
 *    which must own `stream`) looks up the array's device address and fills
 *    the array with 0xFF on `stream`; make that first call before any stream
 *    capture.  Every call that returns FQT1_OK leaves the part it used at
 *    0xFF, as a workspace after fqt1_scq_workspace_init.  A call that returns
 *    an error may leave keys behind, so the next call on that device fills the
 *    array again (one extra fill).  Calls whose work overlaps on the GPU
 *    (concurrent streams) race on the array.
 *  - Allocates nothing: no cudaMalloc / cudaFree or allocating library call.
 * All other arguments, results and errors are those of fqt1_scq_quantize. */
#define FQT1_NOALLOC_SCRATCH_KEYS 16384
fqt1_status fqt1_scq_quantize_noalloc(const float* g, int64_t M, int64_t D, const float* gamma,
                                      const fqt1_agp_params* p_sample, const fqt1_agp_params* p_channel,
                                      fqt1_qgrad* psq, fqt1_qgrad* pcq, int32_t* dev_status, void* stream);

/* grad_input side of SCQ (Eq. 21 with Sec. 5.3's per-sample scales):
 * acc[r, k] = sum_j q[r, j] sign(W)[j, k] over the kept rows r (kept order),
 * dx[m, k] = S'_g acc + Z'_g colsum_w[k] for rows of kept groups, 0 for
 * pruned rows.  sw_col: [K][words(D)]; colsum_w: [K] = sum_j sign(W)[j, k].
 * acc: [capacity * rows_per_group][K] int32 or NULL; dx: [M][K] fp32 or NULL
 * (a convolution passes acc and folds it with fqt1_col2im). */
fqt1_status fqt1_bwd_input_gemm(const fqt1_qgrad* psq, const uint32_t* sw_col, const int32_t* colsum_w, int64_t M,
                                int64_t D, int64_t K, const fqt1_agp_params* p, int32_t* acc, float* dx,
                                void* stream);

/* Folder of App. C on the integer accumulators, then dequantization:
 * dx[n, c, h, w] = S'_n * sum(acc taps) + Z'_n * sum(colsum_w taps) over the
 * taps of the unfolded matrix that read pixel (h, w); pruned samples get 0.
 * acc: [capacity * Ho*Wo][K] from fqt1_bwd_input_gemm; dx: [N, C, H, W]. */
fqt1_status fqt1_col2im(const int32_t* acc, const fqt1_qgrad* psq, const int32_t* colsum_w, int32_t N, int32_t C,
                        int32_t H, int32_t W, int32_t kh, int32_t kw, int32_t stride, int32_t pad, float* dx,
                        void* stream);

/* grad_input of a convolution for any window, stride and map size, as two calls
 * through column-major integer accumulators (Eq. 21 with Sec. 5.3's per-sample
 * scales, App. C Folder).  The first call is fqt1_bwd_input_gemm's integer
 * product with acc stored column-major:
 *   acc[k * ld_acc + r] = sum_j q[r, j] sign(W)[j, k] for the kept rows r (kept
 *   order, r < kept_count * rows_per_group); entries of other rows are not written.
 * acc_bits: 32 (int32) or 16 (int16, exact when (2^bits - 1) * D <= 32767, else
 * FQT1_ERR_INVALID_ARG; it halves the accumulators' traffic).  ld_acc >= capacity
 * * rows_per_group and a multiple of 4 (int32) or 8 (int16); a multiple of 32
 * keeps every column 128-byte aligned.  acc: [K][ld_acc], 16-byte aligned. */
fqt1_status fqt1_bwd_input_gemm_colmajor(const fqt1_qgrad* psq, const uint32_t* sw_col, int64_t M, int64_t D,
                                         int64_t K, const fqt1_agp_params* p, void* acc, int32_t acc_bits,
                                         int64_t ld_acc, void* stream);

/* The same product with sign(W)^T given as e4m3 bytes (+1 = 0x38, -1 = 0xB8, bytes
 * past D zero), wt_e4m3: [K][ld_wt], ld_wt >= fqt1_codes_ld(D) and a multiple of 16
 * (fqt1_binarize_pack_e4m3's transposed output): the B operand then goes to the
 * tensor cores by TMA, unexpanded.  Same acc, bit for bit. */
fqt1_status fqt1_bwd_input_gemm_colmajor_e4m3w(const fqt1_qgrad* psq, const uint8_t* wt_e4m3, int64_t ld_wt,
                                               int64_t M, int64_t D, int64_t K, const fqt1_agp_params* p,
                                               void* acc, int32_t acc_bits, int64_t ld_acc, void* stream);

/* The Folder of App. C on those accumulators, then the per-sample
 * dequantization: the same dx as fqt1_col2im (bit for bit), read with every
 * tap of a warp's 32 consecutive outputs as one contiguous run of a column.
 * acc: [C kh kw][ld_acc] from fqt1_bwd_input_gemm_colmajor with the same acc_bits
 * and ld_acc (the row of output pixel (oh, ow) of kept slot s is s Ho Wo + oh Wo + ow;
 * this call reads rows up to kept count x Ho Wo, which the product's rule ld_acc >=
 * capacity x rows_per_group keeps inside each column; it checks only ld_acc >= Ho Wo); dx:
 * [N, C, H, W], pruned samples 0.  N <= 65535, C H W < 2^31 and C kh kw < 2^31,
 * else FQT1_ERR_UNSUPPORTED. */
fqt1_status fqt1_col2im_colmajor(const void* acc, int32_t acc_bits, int64_t ld_acc, const fqt1_qgrad* psq,
                                 const int32_t* colsum_w,
                                 int32_t N, int32_t C, int32_t H, int32_t W, int32_t kh, int32_t kw, int32_t stride,
                                 int32_t pad, float* dx, void* stream);

/* fqt1_col2im_colmajor with dx channels-last: dx[n, h, w, c] (memory order N, H, W, C),
 * the same values.  Each CTA reads its taps along 32 positions and writes 128-byte runs
 * of channels through shared memory. */
fqt1_status fqt1_col2im_colmajor_nhwc(const void* acc, int32_t acc_bits, int64_t ld_acc, const fqt1_qgrad* psq,
                                      const int32_t* colsum_w, int32_t N, int32_t C, int32_t H, int32_t W,
                                      int32_t kh, int32_t kw, int32_t stride, int32_t pad, float* dx, void* stream);

/* grad_input of a convolution with the Folder fused into the product (Eq. 21 with
 * Sec. 5.3's per-sample scales, App. C Folder): the same dx as fqt1_bwd_input_gemm
 * followed by fqt1_col2im, without the int32 accumulators in memory.  A tile of 128
 * accumulator rows holds whole samples, so this call requires Ho*Wo to divide 128
 * (maps of 8x8, 4x4, 2x2 ... pixels), kh*kw <= 128 and, with cb = floor(128 / (kh kw)),
 * 4 (H W kh kw + cb H W + cb kh kw) + 12 (128 / (Ho Wo)) <= 36864 (its shared-memory
 * tables); other shapes return
 * FQT1_ERR_UNSUPPORTED (use the two-call path).  p->rows_per_group must be Ho*Wo.
 * sw_col: [K = C*kh*kw][words(D)]; colsum_w: [K]; dx: [N, C, H, W] (pruned samples 0). */
fqt1_status fqt1_bwd_input_fold(const fqt1_qgrad* psq, const uint32_t* sw_col, const int32_t* colsum_w, int32_t N,
                                int32_t C, int32_t H, int32_t W, int32_t kh, int32_t kw, int32_t stride, int32_t pad,
                                int64_t D, const fqt1_agp_params* p, float* dx, void* stream);

/* grad_weight side of SCQ (Eq. 21 with Sec. 5.3's per-channel scales):
 * acc[c, k] = sum_m q^c[c, m] sign(X)[m, k] for kept channel slots c,
 * dw[j, k] = S^c'_j acc + Z^c'_j colsum_x[k] for kept channels j, 0 for pruned.
 * sx_col: [K][words(M)]; colsum_x: [K] = sum_m sign(X)[m, k];
 * acc: [capacity][K] int32 (required: the integer result, also the reduction
 * target); dw: [D][K] fp32. */
fqt1_status fqt1_bwd_weight_gemm(const fqt1_qgrad* pcq, const uint32_t* sx_col, const int32_t* colsum_x, int64_t M,
                                 int64_t D, int64_t K, const fqt1_agp_params* p, int32_t* acc, float* dw,
                                 void* ws, size_t ws_bytes, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* FQT1_H */
