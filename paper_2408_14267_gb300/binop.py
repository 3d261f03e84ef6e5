"""binop: 1-bit FQT layers for PyTorch, the layer substitution of Sec. 1
(replace torch.nn.Linear / torch.nn.Conv2d with binop.Linear / binop.Conv2d).

Forward (Sec. 5.1): y = (sign(x) sign(W)^T) (.) Gamma (+ bias), with Gamma a
learnable per-channel scale.  Backward (Eq. 21 with SCQ, Sec. 5.3): the gradient
reaching the binary product, G = gY (.) Gamma, is quantized per sample with AGP
(Sec. 5.2) for the input gradient and per channel for the weight gradient;
    dX = Q_PSQ(G) sign(W),   dW = sign(X)^T Q_PCQ(G),
Gamma and the bias get their exact gradients (libfqt1's fqt1_scale_bias_grad),
and sign() is passed by the straight-through estimator: the identity, or the
clipped form (gradient kept where |x| <= t) when `ste_clip` is set.

Every step runs in libfqt1's kernels through the C-ABI; this module allocates the
buffers of a call with PyTorch and passes pointers.  Each backward draws fresh
seeds for its stochastic rounding and masks from the layer's step counter.
Convolution outputs leave the product as [N, Ho, Wo, D] rows and are returned as a
[N, D, Ho, Wo] view of them.
"""
import torch

from . import fqt1
from .layer import conv_out_hw


class QuantConfig:
    """Gradient quantizer of one layer: bitwidth and selection mode of the sample (PSQ)
    and channel (PCQ) branches, the base seed, and the STE clip threshold (None: identity)."""

    def __init__(self, bits=4, mode=0, bits_c=None, mode_c=None, seed=0, ste_clip=None):
        self.bits_s, self.mode_s = bits, mode
        self.bits_c = bits if bits_c is None else bits_c
        self.mode_c = mode if mode_c is None else mode_c
        self.seed = seed
        self.ste_clip = ste_clip


def _seeds(layer):
    """(PSQ seed, PCQ seed) of the layer's next backward; an explicit pair in layer.next_seeds
    (set by tests) is used once."""
    if layer.next_seeds is not None:
        s = layer.next_seeds
        layer.next_seeds = None
        return s
    layer.step += 1
    base = (layer.qcfg.seed * 0x9E3779B97F4A7C15 + layer.step * 0xD1B54A32D192ED03) & ((1 << 64) - 1)
    return base, base ^ 0x5851F42D4C957F2D


def _packed(rows, cols, dev):
    return torch.empty(rows, fqt1.packed_words(cols), dtype=torch.int32, device=dev)


class _BinaryProduct(torch.autograd.Function):
    """One binary layer: x is [M, K] rows (linear) or the [N, C, H, W] input (convolution)."""

    @staticmethod
    def forward(ctx, x, weight, gamma, bias, layer):
        dev = x.device
        # a channels-last convolution input (32k channels) is read in place: its signs are packed
        # into channel planes, which the Unfolder reads instead of x; otherwise x is made contiguous
        nhwc = (layer.conv is not None and x.dim() == 4 and x.shape[1] % 32 == 0 and not x.is_contiguous()
                and x.is_contiguous(memory_format=torch.channels_last))
        if not nhwc:
            x = x.contiguous()
        D = weight.shape[0]
        w2 = weight.detach().reshape(D, -1).contiguous()
        K = w2.shape[1]
        if layer.conv is None:
            M = x.shape[0]
            rpg = 1
        else:
            N, C, H, W = x.shape
            kh, kw, stride, pad = layer.conv
            Ho, Wo = conv_out_hw(H, W, kh, kw, stride, pad)
            M, rpg = N * Ho * Wo, Ho * Wo
        sw_row, sw_col = _packed(D, K, dev), _packed(K, D, dev)
        cs_w = torch.empty(K, dtype=torch.int32, device=dev)
        fqt1.binarize_pack(w2, D, K, K, sw_row, sw_col, cs_w)
        sx_row, sx_col = _packed(M, K, dev), _packed(K, M, dev)
        cs_x = torch.empty(K, dtype=torch.int32, device=dev)
        if layer.conv is None:
            fqt1.binarize_pack(x.detach(), M, K, K, sx_row, sx_col, cs_x)
        elif nhwc:
            planes = torch.empty(N * C * fqt1.plane_words(H, W), dtype=torch.int32, device=dev)
            fqt1.pack_planes_nhwc(x.detach(), N, C, H, W, planes)
            try:
                fqt1.im2col_planes(planes, N, C, H, W, kh, kw, stride, pad, sx_row, sx_col, cs_x)
            except fqt1.Fqt1Error as e:
                if "UNSUPPORTED" not in str(e):
                    raise
                fqt1.im2col(x.detach().contiguous(), N, C, H, W, kh, kw, stride, pad, sx_row, sx_col, cs_x)
        elif fqt1.unfold_from_planes(N, C, H, W, kh, kw, stride, pad):
            # region tiles: sign-pack x into planes in one pass, the Unfolder then reads bits
            planes = torch.empty(N * C * fqt1.plane_words(H, W), dtype=torch.int32, device=dev)
            fqt1.pack_planes(x.detach(), N, C, H, W, planes)
            fqt1.im2col_planes(planes, N, C, H, W, kh, kw, stride, pad, sx_row, sx_col, cs_x)
        else:
            fqt1.im2col(x.detach(), N, C, H, W, kh, kw, stride, pad, sx_row, sx_col, cs_x)
        g = gamma.detach().contiguous()
        b = None if bias is None else bias.detach().contiguous()
        acc = torch.empty(M, D, dtype=torch.int32, device=dev) if gamma.requires_grad else None
        y = torch.empty(M, D, dtype=torch.float32, device=dev)
        fqt1.fwd_gemm_bias(sx_row, sw_row, M, D, K, g, b, acc, y)
        ctx.layer, ctx.shape = layer, (M, K, D, rpg)
        ctx.in_shape = tuple(x.shape)
        ctx.nhwc = nhwc
        ctx.has_bias = bias is not None
        ctx.save_for_backward(x if layer.qcfg.ste_clip is not None else None,
                              weight if layer.qcfg.ste_clip is not None else None, g, acc, sx_col, cs_x, sw_col, cs_w)
        if layer.conv is None:
            return y
        return y.view(N, Ho, Wo, D).permute(0, 3, 1, 2)

    @staticmethod
    def backward(ctx, gy):
        layer = ctx.layer
        M, K, D, rpg = ctx.shape
        x, weight, g, acc, sx_col, cs_x, sw_col, cs_w = ctx.saved_tensors
        dev = gy.device
        gy2 = (gy if layer.conv is None else gy.permute(0, 2, 3, 1)).contiguous().reshape(M, D).float()
        q = layer.qcfg
        seed_s, seed_c = _seeds(layer)
        p_s = fqt1.AgpParams(q.bits_s, q.mode_s, seed_s, rpg)
        p_c = fqt1.AgpParams(q.bits_c, q.mode_c, seed_c, 1)
        cap_s = fqt1.kept_capacity(M // rpg, q.bits_s, q.mode_s)
        cap_c = fqt1.kept_capacity(D, q.bits_c, q.mode_c)
        psq = fqt1.QGradBuffers(M // rpg, cap_s, cap_s * rpg, D, dev)
        pcq = fqt1.QGradBuffers(D, cap_c, cap_c, M, dev)
        ws = fqt1.scq_workspace(M, D, K, rpg, dev)
        status = torch.zeros(4, dtype=torch.int32, device=dev)
        fqt1.scq_quantize(gy2, M, D, g, p_s, p_c, psq, pcq, ws, status)
        dx = dw = dgamma = dbias = None
        if ctx.needs_input_grad[0]:
            if layer.conv is None:
                dx = torch.empty(M, K, dtype=torch.float32, device=dev)
                fqt1.bwd_input_gemm(psq, sw_col, cs_w, M, D, K, p_s, None, dx)
            else:
                N, C, H, W = ctx.in_shape
                kh, kw, stride, pad = layer.conv
                Ho, Wo = conv_out_hw(H, W, kh, kw, stride, pad)
                # a channels-last input gets its gradient channels-last too (returned as an NCHW
                # view of NHWC memory), so that the layers before it need no layout copy
                nhwc = ctx.nhwc
                dx = torch.empty((N, H, W, C) if nhwc else (N, C, H, W), dtype=torch.float32, device=dev)
                if fqt1.fold_supported(Ho, Wo, kh, kw, H, W):
                    fqt1.bwd_input_fold(psq, sw_col, cs_w, N, C, H, W, kh, kw, stride, pad, D, p_s, dx, nhwc=nhwc)
                else:
                    # column-major accumulators (int16 where every sum fits): the Folder reads
                    # every tap as contiguous runs of a column; dx in the input's memory order
                    ld = (max(cap_s * rpg, 1) + 31) // 32 * 32
                    acc_t = torch.int16 if fqt1.colmajor_acc_bits(q.bits_s, D) == 16 else torch.int32
                    acc_cm = torch.empty(K, ld, dtype=acc_t, device=dev)
                    fqt1.bwd_input_gemm_colmajor(psq, sw_col, M, D, K, p_s, acc_cm)
                    fqt1.col2im_colmajor(acc_cm, psq, cs_w, N, C, H, W, kh, kw, stride, pad, dx, nhwc=nhwc)
                if nhwc:
                    dx = dx.permute(0, 3, 1, 2)
            if q.ste_clip is not None:  # x and dx elementwise in the same memory order
                if dx.is_contiguous():
                    fqt1.ste_clip(x.contiguous(), dx, dx.numel(), q.ste_clip)
                else:  # channels-last dx: x in the same order
                    xm = x.contiguous(memory_format=torch.channels_last)
                    fqt1.ste_clip(xm.permute(0, 2, 3, 1).contiguous(), dx.permute(0, 2, 3, 1), dx.numel(),
                                  q.ste_clip)
        if ctx.needs_input_grad[1]:
            acc_dw = torch.empty(max(cap_c, 1), K, dtype=torch.int32, device=dev)
            dw = torch.empty(D, K, dtype=torch.float32, device=dev)
            fqt1.bwd_weight_gemm(pcq, sx_col, cs_x, M, D, K, p_c, acc_dw, dw)
            if q.ste_clip is not None:
                fqt1.ste_clip(weight.detach().reshape(D, K).contiguous(), dw, dw.numel(), q.ste_clip)
            dw = dw.view(layer.weight.shape)
        want_g = ctx.needs_input_grad[2]
        want_b = ctx.has_bias and ctx.needs_input_grad[3]
        if want_g or want_b:
            sb_ws = torch.empty(fqt1.scale_bias_workspace(M, D), dtype=torch.uint8, device=dev)
            dgamma = torch.empty(D, dtype=torch.float32, device=dev) if want_g else None
            dbias = torch.empty(D, dtype=torch.float32, device=dev) if want_b else None
            fqt1.scale_bias_grad(gy2, acc if want_g else None, M, D, dgamma, dbias, sb_ws)
        layer.last_status = status
        return dx, dw, dgamma, dbias, None


class _BinaryLayer(torch.nn.Module):
    def __init__(self, weight_shape, bias, qcfg, device):
        super().__init__()
        D = weight_shape[0]
        fan_in = 1
        for s in weight_shape[1:]:
            fan_in *= s
        self.weight = torch.nn.Parameter(torch.randn(*weight_shape, device=device) * (2.0 / fan_in) ** 0.5)
        self.gamma = torch.nn.Parameter(torch.ones(D, device=device))
        self.bias = torch.nn.Parameter(torch.zeros(D, device=device)) if bias else None
        self.qcfg = qcfg if qcfg is not None else QuantConfig()
        self.step = 0
        self.next_seeds = None
        self.last_status = None

    def nonfinite_gradient(self):
        """True if the last backward met a non-finite gradient value (reads the device flag)."""
        return self.last_status is not None and bool(int(self.last_status[0].item()) & 1)


class Linear(_BinaryLayer):
    """y = (sign(x) sign(W)^T) (.) Gamma (+ bias) for x [N, in_features]; 1-bit FQT backward."""

    def __init__(self, in_features, out_features, bias=False, qcfg=None, device="cuda"):
        super().__init__((out_features, in_features), bias, qcfg, device)
        self.conv = None

    def forward(self, x):
        return _BinaryProduct.apply(x, self.weight, self.gamma, self.bias, self)


class Conv2d(_BinaryLayer):
    """Binary convolution: y = Unfolder(sign(x)) sign(W)^T (.) Gamma (+ bias), NCHW in and out."""

    def __init__(self, in_channels, out_channels, kernel_size, stride=1, padding=0, bias=False, qcfg=None,
                 device="cuda"):
        k = kernel_size if isinstance(kernel_size, tuple) else (kernel_size, kernel_size)
        super().__init__((out_channels, in_channels, k[0], k[1]), bias, qcfg, device)
        self.conv = (k[0], k[1], stride, padding)

    def forward(self, x):
        return _BinaryProduct.apply(x, self.weight, self.gamma, self.bias, self)
