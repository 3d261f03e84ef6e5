"""ctypes binding of libfqt1 (argument marshalling only).

Every function here forwards device pointers and sizes to the C-ABI entry
point of the same name declared in include/fqt1.h; all arithmetic runs in the
library's CUDA kernels.  PyTorch supplies device memory and streams.  There is
no fallback: if libfqt1.so is missing or a call fails, an exception is raised.
"""
import ctypes as C
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libfqt1.so")

SYSTEMATIC, BERNOULLI, TOPK = 0, 1, 2
DEV_NONFINITE, DEV_TIMEOUT = 0x100, 0x200
STATUS_NAMES = {0: "FQT1_OK", 1: "FQT1_ERR_INVALID_ARG", 2: "FQT1_ERR_MISALIGNED", 3: "FQT1_ERR_UNSUPPORTED",
                4: "FQT1_ERR_WORKSPACE", 5: "FQT1_ERR_CUDA"}


class AgpParams(C.Structure):
    _fields_ = [("bits", C.c_int32), ("mode", C.c_int32), ("seed", C.c_uint64), ("rows_per_group", C.c_int64)]


class QGrad(C.Structure):
    _fields_ = [("group_min", C.c_void_p), ("group_range", C.c_void_p), ("p_hat", C.c_void_p),
                ("slot_of_group", C.c_void_p), ("kept_idx", C.c_void_p), ("kept_count", C.c_void_p),
                ("scale", C.c_void_p), ("zero", C.c_void_p), ("codes", C.c_void_p), ("ld_codes", C.c_int64)]


class Fqt1Error(RuntimeError):
    pass


_lib = None
_VP, _I64, _I32 = C.c_void_p, C.c_int64, C.c_int32
_SIGS = {
    "fqt1_packed_words": (_I64, [_I64]),
    "fqt1_kept_capacity": (_I64, [_I64, _I32, _I32]),
    "fqt1_codes_ld": (_I64, [_I64]),
    "fqt1_workspace_size": (C.c_size_t, [_I32, _I64, _I64, _I64, _I32]),
    "fqt1_last_cuda_error": (C.c_char_p, []),
    "fqt1_kernel_launches": (_I64, []),
    "fqt1_binarize_pack": (C.c_int, [_VP, _I64, _I64, _I64, _VP, _VP, _VP, _VP]),
    "fqt1_im2col": (C.c_int, [_VP] + [_I32] * 8 + [_VP, _VP, _VP, _VP]),
    "fqt1_fwd_gemm": (C.c_int, [_VP, _VP, _I64, _I64, _I64, _VP, _VP, _VP, _VP]),
    "fqt1_fwd_gemm_bias": (C.c_int, [_VP, _VP, _I64, _I64, _I64, _VP, _VP, _VP, _VP, _VP]),
    "fqt1_test_expired_wait": (C.c_int, [_VP, _VP, _I64, _I64, _I64, _VP, _VP, _VP, _VP]),
    "fqt1_scale_bias_workspace": (C.c_size_t, [_I64, _I64]),
    "fqt1_scale_bias_grad": (C.c_int, [_VP, _VP, _I64, _I64, _VP, _VP, _VP, C.c_size_t, _VP]),
    "fqt1_ste_clip": (C.c_int, [_VP, _VP, _I64, C.c_float, _VP]),
    "fqt1_agp_quantize_grad": (C.c_int, [_VP, _I64, _I64, _I32, _VP, _VP, _VP, _VP, C.c_size_t, _VP, _VP]),
    "fqt1_scq_workspace_init": (C.c_int, [_VP, C.c_size_t, _VP]),
    "fqt1_expand_signs_e4m3": (C.c_int, [_VP, _I64, _I64, _VP, _I64, _VP]),
    "fqt1_binarize_pack_e4m3": (C.c_int, [_VP, _I64, _I64, _I64, _VP, _VP, _VP, _VP, _I64, _VP, _I64, _VP]),
    "fqt1_fwd_gemm_e4m3w": (C.c_int, [_VP, _VP, _I64, _I64, _I64, _I64, _VP, _VP, _VP, _VP, _VP]),
    "fqt1_bwd_input_fold_e4m3w": (C.c_int, [_VP, _VP, _I64, _VP] + [_I32] * 8 + [_I64, _VP, _VP, _VP]),
    "fqt1_im2col_e4m3": (C.c_int, [_VP] + [_I32] * 8 + [_VP, _I64, _VP, _I64, _VP, _VP]),
    "fqt1_fwd_gemm_e4m3x": (C.c_int, [_VP, _I64, _VP, _I64, _I64, _I64, _I64, _VP, _VP, _VP, _VP, _VP]),
    "fqt1_bwd_weight_gemm_e4m3x": (C.c_int, [_VP, _VP, _I64, _VP, _I64, _I64, _I64, _VP, _VP, _VP, _VP]),
    "fqt1_pack_pixels": (C.c_int, [_VP, _I32, _I32, _I32, _I32, _VP, _VP]),
    "fqt1_pack_planes_nhwc": (C.c_int, [_VP, _I32, _I32, _I32, _I32, _VP, _VP]),
    "fqt1_pack_planes": (C.c_int, [_VP, _I32, _I32, _I32, _I32, _VP, _VP]),
    "fqt1_im2col_path": (_I32, [_I32] * 8),
    "fqt1_im2col_planes": (C.c_int, [_VP] + [_I32] * 8 + [_VP, _VP, _VP, _VP]),
    "fqt1_pack_weight_taps": (C.c_int, [_VP, _I64, _I32, _I32, _I32, _VP, _VP]),
    "fqt1_conv_implicit_supported": (_I32, [_I32] * 8),
    "fqt1_conv_fwd_implicit": (C.c_int, [_VP, _VP] + [_I32] * 8 + [_I64, _VP, _VP, _VP, _VP, _VP]),
    "fqt1_scq_quantize": (C.c_int, [_VP, _I64, _I64, _VP, _VP, _VP, _VP, _VP, _VP, C.c_size_t, _VP, _VP]),
    "fqt1_scq_quantize_noalloc": (C.c_int, [_VP, _I64, _I64, _VP, _VP, _VP, _VP, _VP, _VP, _VP]),
    "fqt1_bwd_input_gemm": (C.c_int, [_VP, _VP, _VP, _I64, _I64, _I64, _VP, _VP, _VP, _VP]),
    "fqt1_col2im": (C.c_int, [_VP, _VP, _VP] + [_I32] * 8 + [_VP, _VP]),
    "fqt1_bwd_input_gemm_colmajor": (C.c_int, [_VP, _VP, _I64, _I64, _I64, _VP, _VP, _I32, _I64, _VP]),
    "fqt1_col2im_colmajor": (C.c_int, [_VP, _I32, _I64, _VP, _VP] + [_I32] * 8 + [_VP, _VP]),
    "fqt1_col2im_colmajor_nhwc": (C.c_int, [_VP, _I32, _I64, _VP, _VP] + [_I32] * 8 + [_VP, _VP]),
    "fqt1_bwd_input_gemm_colmajor_e4m3w": (C.c_int, [_VP, _VP, _I64, _I64, _I64, _I64, _VP, _VP, _I32, _I64,
                                                     _VP]),
    "fqt1_col2im_nhwc": (C.c_int, [_VP, _VP, _VP] + [_I32] * 8 + [_VP, _VP]),
    "fqt1_bwd_input_fold_nhwc": (C.c_int, [_VP, _VP, _VP] + [_I32] * 8 + [_I64, _VP, _VP, _VP]),
    "fqt1_bwd_input_fold": (C.c_int, [_VP, _VP, _VP] + [_I32] * 8 + [_I64, _VP, _VP, _VP]),
    "fqt1_bwd_weight_gemm": (C.c_int, [_VP, _VP, _VP, _I64, _I64, _I64, _VP, _VP, _VP, _VP, C.c_size_t, _VP]),
}


def lib():
    """Load libfqt1.so (built by paper_2408_14267_gb300.build)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise Fqt1Error(f"{LIB_PATH} is missing: build it with paper_2408_14267_gb300.build.build()")
        L = C.CDLL(LIB_PATH)
        for name, (res, args) in _SIGS.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def exported_names():
    return list(_SIGS)


def _check(status, name):
    if status != 0:
        msg = STATUS_NAMES.get(status, str(status))
        if status == 5:
            msg += " (" + lib().fqt1_last_cuda_error().decode() + ")"
        raise Fqt1Error(f"{name} failed: {msg}")


def _p(t):
    """Device pointer of a CUDA tensor, or None."""
    if t is None:
        return None
    if not t.is_cuda:
        raise Fqt1Error("libfqt1 takes CUDA tensors only")
    return t.data_ptr()


def _s(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return C.c_void_p(stream.cuda_stream)


# ----------------------------------------------------------------- helpers
def packed_words(n):
    return lib().fqt1_packed_words(n)


def kept_capacity(n, bits, mode):
    return lib().fqt1_kept_capacity(n, bits, mode)


def codes_ld(n):
    return lib().fqt1_codes_ld(n)


def kernel_launches():
    return lib().fqt1_kernel_launches()


def workspace_size(which, M, D, K, rows_per_group):
    return lib().fqt1_workspace_size(which, M, D, K, rows_per_group)


def scq_workspace(M, D, K, rows_per_group, device, stream=None):
    """A workspace of fqt1_agp_quantize_grad / fqt1_scq_quantize, filled with 0xFF by
    fqt1_scq_workspace_init; the calls leave it so, and it can be reused for any shape it fits."""
    import torch
    ws = torch.empty(workspace_size(0, M, D, K, rows_per_group), dtype=torch.uint8, device=device)
    scq_workspace_init(ws, stream)
    return ws


def scq_workspace_init(ws, stream=None):
    _check(lib().fqt1_scq_workspace_init(_p(ws), ws.numel() * ws.element_size(), _s(stream)),
           "fqt1_scq_workspace_init")


# ------------------------------------------------------------ entry points
def binarize_pack(x, rows, cols, ld, row_bits=None, col_bits=None, colsum=None, stream=None):
    _check(lib().fqt1_binarize_pack(_p(x), rows, cols, ld, _p(row_bits), _p(col_bits), _p(colsum), _s(stream)),
           "fqt1_binarize_pack")


def im2col(x, N, Cin, H, W, kh, kw, stride, pad, row_bits=None, col_bits=None, colsum=None, stream=None):
    _check(lib().fqt1_im2col(_p(x), N, Cin, H, W, kh, kw, stride, pad, _p(row_bits), _p(col_bits), _p(colsum),
                             _s(stream)), "fqt1_im2col")


def test_expired_wait(sx_row, sw_row, M, D, K, gamma, y, dev_status, stream=None):
    _check(lib().fqt1_test_expired_wait(_p(sx_row), _p(sw_row), M, D, K, _p(gamma), _p(y), _p(dev_status),
                                        _s(stream)), "fqt1_test_expired_wait")


def fwd_gemm(sx_row, sw_row, M, D, K, gamma, acc, y, stream=None):
    _check(lib().fqt1_fwd_gemm(_p(sx_row), _p(sw_row), M, D, K, _p(gamma), _p(acc), _p(y), _s(stream)),
           "fqt1_fwd_gemm")


def expand_signs_e4m3(bits, rows, n, out, stream=None):
    _check(lib().fqt1_expand_signs_e4m3(_p(bits), rows, n, _p(out), out.shape[-1], _s(stream)),
           "fqt1_expand_signs_e4m3")


def binarize_pack_e4m3(x, rows, cols, ld, row_bits, col_bits, colsum, row_e4m3, col_e4m3, stream=None):
    _check(lib().fqt1_binarize_pack_e4m3(_p(x), rows, cols, ld, _p(row_bits), _p(col_bits), _p(colsum), _p(row_e4m3),
                                         row_e4m3.shape[-1] if row_e4m3 is not None else 0, _p(col_e4m3),
                                         col_e4m3.shape[-1] if col_e4m3 is not None else 0, _s(stream)),
           "fqt1_binarize_pack_e4m3")


def im2col_e4m3(x, N, Cin, H, W, kh, kw, stride, pad, x_row=None, x_col=None, colsum=None, stream=None):
    _check(lib().fqt1_im2col_e4m3(_p(x), N, Cin, H, W, kh, kw, stride, pad, _p(x_row),
                                  0 if x_row is None else x_row.shape[-1], _p(x_col),
                                  0 if x_col is None else x_col.shape[-1], _p(colsum), _s(stream)),
           "fqt1_im2col_e4m3")


def fwd_gemm_e4m3x(x_e4m3, w_e4m3, M, D, K, gamma, bias, acc, y, stream=None):
    _check(lib().fqt1_fwd_gemm_e4m3x(_p(x_e4m3), x_e4m3.shape[-1], _p(w_e4m3), w_e4m3.shape[-1], M, D, K, _p(gamma),
                                     _p(bias), _p(acc), _p(y), _s(stream)), "fqt1_fwd_gemm_e4m3x")


def bwd_weight_gemm_e4m3x(pcq, x_col_e4m3, colsum_x, M, D, K, params, acc, dw, stream=None):
    _check(lib().fqt1_bwd_weight_gemm_e4m3x(C.byref(pcq.c), _p(x_col_e4m3), x_col_e4m3.shape[-1], _p(colsum_x), M, D,
                                            K, C.byref(params), _p(acc), _p(dw), _s(stream)),
           "fqt1_bwd_weight_gemm_e4m3x")


def fwd_gemm_e4m3w(sx_row, w_e4m3, M, D, K, gamma, bias, acc, y, stream=None):
    _check(lib().fqt1_fwd_gemm_e4m3w(_p(sx_row), _p(w_e4m3), w_e4m3.shape[-1], M, D, K, _p(gamma), _p(bias),
                                     _p(acc), _p(y), _s(stream)), "fqt1_fwd_gemm_e4m3w")


def bwd_input_fold_e4m3w(psq, wt_e4m3, colsum_w, N, Cin, H, W, kh, kw, stride, pad, D, p, dx, stream=None):
    _check(lib().fqt1_bwd_input_fold_e4m3w(C.byref(psq.c), _p(wt_e4m3), wt_e4m3.shape[-1], _p(colsum_w), N, Cin, H,
                                           W, kh, kw, stride, pad, D, C.byref(p), _p(dx), _s(stream)),
           "fqt1_bwd_input_fold_e4m3w")


def plane_words(H, W):
    return (H * W + 31) // 32


def pack_planes(x, N, Cin, H, W, planes, stream=None):
    _check(lib().fqt1_pack_planes(_p(x), N, Cin, H, W, _p(planes), _s(stream)), "fqt1_pack_planes")


def im2col_path(N, Cin, H, W, kh, kw, stride, pad):
    """2: whole-image tiles from x; 1: region tiles (planes first read 32x fewer bytes); 0: gather."""
    return lib().fqt1_im2col_path(N, Cin, H, W, kh, kw, stride, pad)


def unfold_from_planes(N, Cin, H, W, kh, kw, stride, pad):
    """Whether a contiguous x is sign-packed into planes before the Unfolder: every region-tile
    shape (im2col_path 1).  Reading x directly is faster for the Unfolder alone on 4 x 4, 2 x 2
    and 7 x 7 maps (eager, L2 flushed: 19-24 us against 27-31 us for the two launches), but not
    for the three-branch layer step: on the 4 x 4 VGG-16 layers three same-GPU sweeps gave 209.5
    and 220.3 us (direct) against 206.9 us (planes first) for conv8-conv10, single replays
    spreading over 66-86 us with the order in which the concurrent branches get their SMs."""
    return im2col_path(N, Cin, H, W, kh, kw, stride, pad) == 1


def pack_planes_nhwc(x, N, Cin, H, W, planes, stream=None):
    _check(lib().fqt1_pack_planes_nhwc(_p(x), N, Cin, H, W, _p(planes), _s(stream)), "fqt1_pack_planes_nhwc")


def im2col_planes(planes, N, Cin, H, W, kh, kw, stride, pad, row_bits=None, col_bits=None, colsum=None, stream=None):
    _check(lib().fqt1_im2col_planes(_p(planes), N, Cin, H, W, kh, kw, stride, pad, _p(row_bits), _p(col_bits),
                                    _p(colsum), _s(stream)), "fqt1_im2col_planes")


def pack_pixels(x, N, Cin, H, W, x_pix, stream=None):
    _check(lib().fqt1_pack_pixels(_p(x), N, Cin, H, W, _p(x_pix), _s(stream)), "fqt1_pack_pixels")


def pack_weight_taps(w, D, Cin, kh, kw, w_taps, stream=None):
    _check(lib().fqt1_pack_weight_taps(_p(w), D, Cin, kh, kw, _p(w_taps), _s(stream)), "fqt1_pack_weight_taps")


def conv_implicit_supported(N, Cin, H, W, kh, kw, stride, pad):
    return bool(lib().fqt1_conv_implicit_supported(N, Cin, H, W, kh, kw, stride, pad))


def conv_fwd_implicit(x_pix, w_taps, N, Cin, H, W, kh, kw, stride, pad, D, gamma, bias, acc, y, stream=None):
    _check(lib().fqt1_conv_fwd_implicit(_p(x_pix), _p(w_taps), N, Cin, H, W, kh, kw, stride, pad, D, _p(gamma),
                                        _p(bias), _p(acc), _p(y), _s(stream)), "fqt1_conv_fwd_implicit")


def fwd_gemm_bias(sx_row, sw_row, M, D, K, gamma, bias, acc, y, stream=None):
    _check(lib().fqt1_fwd_gemm_bias(_p(sx_row), _p(sw_row), M, D, K, _p(gamma), _p(bias), _p(acc), _p(y),
                                    _s(stream)), "fqt1_fwd_gemm_bias")


def scale_bias_workspace(M, D):
    return lib().fqt1_scale_bias_workspace(M, D)


def scale_bias_grad(gy, acc, M, D, dgamma, dbias, ws, stream=None):
    _check(lib().fqt1_scale_bias_grad(_p(gy), _p(acc), M, D, _p(dgamma), _p(dbias), _p(ws),
                                      ws.numel() * ws.element_size(), _s(stream)), "fqt1_scale_bias_grad")


def ste_clip(x, dx, n, t, stream=None):
    _check(lib().fqt1_ste_clip(_p(x), _p(dx), n, float(t), _s(stream)), "fqt1_ste_clip")


def agp_quantize_grad(g, M, D, group_axis, gamma, params, qgrad, ws, dev_status, stream=None):
    _check(lib().fqt1_agp_quantize_grad(_p(g), M, D, group_axis, _p(gamma), C.byref(params), C.byref(qgrad.c),
                                        _p(ws), ws.numel() * ws.element_size(), _p(dev_status), _s(stream)),
           "fqt1_agp_quantize_grad")


def scq_quantize(g, M, D, gamma, p_sample, p_channel, psq, pcq, ws, dev_status, stream=None):
    _check(lib().fqt1_scq_quantize(_p(g), M, D, _p(gamma), C.byref(p_sample), C.byref(p_channel), C.byref(psq.c),
                                   C.byref(pcq.c), _p(ws), ws.numel() * ws.element_size(), _p(dev_status),
                                   _s(stream)), "fqt1_scq_quantize")


def scq_quantize_noalloc(g, M, D, gamma, p_sample, p_channel, psq, pcq, dev_status, stream=None):
    """fqt1_scq_quantize without a workspace argument: the scratch is a fixed array inside
    the library, for callers that cannot allocate device memory at this point."""
    _check(lib().fqt1_scq_quantize_noalloc(_p(g), M, D, _p(gamma), C.byref(p_sample), C.byref(p_channel),
                                           C.byref(psq.c), C.byref(pcq.c), _p(dev_status), _s(stream)),
           "fqt1_scq_quantize_noalloc")


def bwd_input_gemm(psq, sw_col, colsum_w, M, D, K, params, acc, dx, stream=None):
    _check(lib().fqt1_bwd_input_gemm(C.byref(psq.c), _p(sw_col), _p(colsum_w), M, D, K, C.byref(params), _p(acc),
                                     _p(dx), _s(stream)), "fqt1_bwd_input_gemm")


def col2im(acc, psq, colsum_w, N, Cin, H, W, kh, kw, stride, pad, dx, stream=None, nhwc=False):
    fn = lib().fqt1_col2im_nhwc if nhwc else lib().fqt1_col2im
    _check(fn(_p(acc), C.byref(psq.c), _p(colsum_w), N, Cin, H, W, kh, kw, stride, pad, _p(dx), _s(stream)),
           "fqt1_col2im_nhwc" if nhwc else "fqt1_col2im")


def _acc_bits(acc):
    return {torch.int16: 16, torch.int32: 32}[acc.dtype]


def bwd_input_gemm_colmajor(psq, sw_col, M, D, K, params, acc, stream=None):
    """acc: [K][ld] int32 or int16 (its dtype selects the accumulator width)."""
    _check(lib().fqt1_bwd_input_gemm_colmajor(C.byref(psq.c), _p(sw_col), M, D, K, C.byref(params), _p(acc),
                                              _acc_bits(acc), acc.shape[1], _s(stream)),
           "fqt1_bwd_input_gemm_colmajor")


def bwd_input_gemm_colmajor_e4m3w(psq, wt8, M, D, K, params, acc, stream=None):
    _check(lib().fqt1_bwd_input_gemm_colmajor_e4m3w(C.byref(psq.c), _p(wt8), wt8.shape[1], M, D, K, C.byref(params),
                                                    _p(acc), _acc_bits(acc), acc.shape[1], _s(stream)),
           "fqt1_bwd_input_gemm_colmajor_e4m3w")


def col2im_colmajor(acc, psq, colsum_w, N, Cin, H, W, kh, kw, stride, pad, dx, stream=None, nhwc=False):
    fn = lib().fqt1_col2im_colmajor_nhwc if nhwc else lib().fqt1_col2im_colmajor
    _check(fn(_p(acc), _acc_bits(acc), acc.shape[1], C.byref(psq.c), _p(colsum_w), N, Cin, H, W, kh, kw, stride, pad,
              _p(dx), _s(stream)), "fqt1_col2im_colmajor_nhwc" if nhwc else "fqt1_col2im_colmajor")


def colmajor_acc_bits(bits, D):
    """16 when every grad_input accumulator fits int16 ((2^bits - 1) D <= 32767), else 32."""
    return 16 if ((1 << bits) - 1) * D <= 32767 else 32


def bwd_input_fold(psq, sw_col, colsum_w, N, Cin, H, W, kh, kw, stride, pad, D, params, dx, stream=None,
                   nhwc=False):
    fn = lib().fqt1_bwd_input_fold_nhwc if nhwc else lib().fqt1_bwd_input_fold
    _check(fn(C.byref(psq.c), _p(sw_col), _p(colsum_w), N, Cin, H, W, kh, kw, stride, pad, D, C.byref(params),
              _p(dx), _s(stream)), "fqt1_bwd_input_fold_nhwc" if nhwc else "fqt1_bwd_input_fold")


def fold_supported(Ho, Wo, kh, kw, H, W):
    """The fused grad_input + Folder needs whole samples per 128-row tile (Ho*Wo divides 128)."""
    if 128 % (Ho * Wo) != 0 or kh * kw > 128:
        return False
    khw = kh * kw
    cb = 128 // khw
    return 4 * (H * W * khw + cb * H * W + cb * khw) + 12 * (128 // (Ho * Wo)) <= 36864


def bwd_weight_gemm(pcq, sx_col, colsum_x, M, D, K, params, acc, dw, ws=None, stream=None):
    nbytes = 0 if ws is None else ws.numel() * ws.element_size()
    _check(lib().fqt1_bwd_weight_gemm(C.byref(pcq.c), _p(sx_col), _p(colsum_x), M, D, K, C.byref(params), _p(acc),
                                      _p(dw), _p(ws), nbytes, _s(stream)), "fqt1_bwd_weight_gemm")


# --------------------------------------------------------- buffer holders
class QGradBuffers:
    """Device arrays of one fqt1_qgrad branch (n groups, `rows` code rows of `row_len` codes)."""

    def __init__(self, n, capacity, code_rows, row_len, device="cuda"):
        f = dict(device=device)
        self.n, self.capacity = n, capacity
        self.group_min = torch.empty(n, dtype=torch.float32, **f)
        self.group_range = torch.empty(n, dtype=torch.float32, **f)
        self.p_hat = torch.empty(n, dtype=torch.float64, **f)
        self.slot_of_group = torch.empty(n, dtype=torch.int32, **f)
        self.kept_idx = torch.empty(max(capacity, 1), dtype=torch.int32, **f)
        self.kept_count = torch.zeros(4, dtype=torch.int32, **f)
        self.scale = torch.empty(max(capacity, 1), dtype=torch.float32, **f)
        self.zero = torch.empty(max(capacity, 1), dtype=torch.float32, **f)
        self.ld = codes_ld(row_len)
        self.codes = torch.zeros(max(code_rows, 1), self.ld, dtype=torch.uint8, **f)
        self.c = QGrad(_p(self.group_min), _p(self.group_range), _p(self.p_hat), _p(self.slot_of_group),
                       _p(self.kept_idx), _p(self.kept_count), _p(self.scale), _p(self.zero), _p(self.codes),
                       self.ld)

    def count(self):
        return int(self.kept_count[0].item())
