"""Plain CPU oracle of one 1-bit FQT layer step (1-Bit FQT, arXiv 2408.14267).

TEST INFRASTRUCTURE.  Only `tests/`, `__graft_entry__.smoke()` and the
CPU-baseline / reference leg of `bench.py` may import this module.  It shares
no code with the CUDA library and is never on the product path.

Every function works on logical (unpadded) numpy arrays and follows the
paper's steps in its own order and notation:

* forward, Sec. 5.1: sign(x) = -1 if x <= 0 else +1, H = (sign(H) sign(Theta)) (.) Gamma
* unbiased range quantizer, Sec. 3.2: B = 2^b - 1, Z = min, R = max - min,
  q = SR(B (x - Z) / R), dequantized as q R / B + Z
* AGP, Sec. 5.2: per-group ranges, keep probabilities p_i with sum n/b and
  p_i proportional to R_i, masks m_i with E[m_i / p_i] = 1, Q_g = Q_PSQ^b(M grad)
* SCQ, Sec. 5.3: per-sample scales for the input gradient, per-channel scales
  for the weight gradient; both scales factor out of the integer products
* bit-plane form and the {0,1} -> {-1,+1} conversion, App. C
* Unfolder / Folder for convolutions, App. C

Where the paper is silent the oracle takes these readings (each is listed with
its reason in the design notes of the repository):

R1  zero padding of a convolution contributes x = 0, i.e. sign -1.
R2  Gamma is an input vector of length D; the gradient reaching the binary
    product is G = gY (.) Gamma (fp32 multiply), because a per-channel Gamma
    lies along the contraction dimension of grad_input.
R3  keep probabilities are water-filled: p_i = min(1, c R_i) with sum n/b,
    computed exactly in fixed point (see `agp_probabilities`).  This meets the
    three conditions of Sec. 5.2 and equals p_i = n R_i / (b R_total) whenever
    no probability exceeds 1.  b = 1 keeps every group (plain PSQ/PCQ).
R4  masks: SYSTEMATIC (default) draws one uniform offset and keeps group i iff
    a multiple of 2^32 falls in its slot of the cumulative sum of
    P_i = floor(p_i 2^32); each group is kept with probability exactly
    p^_i = P_i 2^-32 and the kept count is floor or ceil of sum p^.
    BERNOULLI keeps each group independently with probability p^_i.
    TOPK keeps the floor(n/b) largest ranges with p^ = 1 (App. B analysis, biased).
R5  stochastic rounding in fp32: inv = B / R, t = (x - Z) * inv, q = floor(t)
    + [u < t - floor(t)], u = (w >> 8) 2^-24 with w a Philox word, q clamped
    to [0, B]; groups with R = 0 (or B / R not finite) get q = 0.  The word of
    element (m, j) is number m*D + j of stream 0 for PSQ (row-major) and number
    j*M + m of stream 1 for PCQ (column-major).  Codes do not depend on p; p
    enters the scale S' = R / (B p^) and zero point Z' = Z / p^.
R6  dequantization is fp32: a = S' * float(acc), c = Z' * float(colsum),
    out = a + c; pruned rows / channels are exactly 0.
R10 a layer may add a per-channel bias after the scale (y = Gamma * acc + bias,
    fp32 multiply then add); the gradients of Gamma and of the bias are the
    exact sums over the rows of gY * acc and gY (float64 here).  The
    straight-through estimator of sign() is the identity; its clipped form
    keeps the gradient where |x| <= t.
"""
import numpy as np

from .philox import uniform_u32

SYSTEMATIC, BERNOULLI, TOPK = 0, 1, 2
STREAM_SR_PSQ, STREAM_SR_PCQ, STREAM_SEL_SAMPLE, STREAM_SEL_CHANNEL = 0, 1, 2, 3
FIXED_POINT_BITS = 40
TWO32 = 1 << 32

f32 = np.float32


# --------------------------------------------------------------------------
# Forward: binarization and the binary product (Sec. 5.1, App. C)
# --------------------------------------------------------------------------
def sign(x):
    """Deterministic forward quantizer of Sec. 5.1: +1 iff x > 0, else -1."""
    return np.where(np.asarray(x) > 0, 1, -1).astype(np.int8)


def int_matmul(a, b_t):
    """Exact integer product a @ b_t.T of small-integer matrices.

    Every product and partial sum is an integer below 2^53, so the float64
    matrix product is exact whatever its summation order.
    """
    r = np.asarray(a, dtype=np.float64) @ np.asarray(b_t, dtype=np.float64).T
    return r.astype(np.int64)


def forward(x_u, w, gamma):
    """Binarized forward of a fully connected layer (Sec. 5.1).

    x_u [M, K] fp32, w [D, K] fp32, gamma [D] fp32 (None: Gamma = 1).
    Returns (acc int64 [M, D] = sign(x_u) sign(w)^T, y fp32 = gamma_j * acc).
    """
    acc = int_matmul(sign(x_u), sign(w))
    if gamma is None:  # no Gamma: unit scale
        return acc, acc.astype(f32)
    y = (np.asarray(gamma, dtype=f32)[None, :] * acc.astype(f32)).astype(f32)
    return acc, y


def forward_bias(x_u, w, gamma, bias):
    """Forward of Sec. 5.1 with a per-channel bias after the scale (reading R10):
    y = fp32(Gamma * acc) + bias, both operations rounded to fp32."""
    acc, y = forward(x_u, w, gamma)
    if bias is None:
        return acc, y
    return acc, (y + np.asarray(bias, dtype=f32)[None, :]).astype(f32)


def scale_bias_grad(gy, acc):
    """Gradients of the layer's learnable scale Gamma (Sec. 5.1, y = acc (.) Gamma) and of
    its bias (reading R10): dGamma_j = sum_m gY[m, j] acc[m, j], dbias_j = sum_m gY[m, j],
    in float64."""
    g = np.asarray(gy, dtype=np.float64)
    return (g * np.asarray(acc, dtype=np.float64)).sum(axis=0), g.sum(axis=0)


def ste_clip(x, dx, t=1.0):
    """Clipped straight-through estimator of sign() (reading R10): the gradient passes
    where |x| <= t and is 0 elsewhere (also where x is NaN)."""
    x = np.asarray(x)
    return np.where(np.abs(x) <= t, dx, 0).astype(np.asarray(dx).dtype)


def colsum_sign(a):
    """Column sums of sign(a): the colsum terms of the SCQ dequantization."""
    return sign(a).astype(np.int64).sum(axis=0)


# --------------------------------------------------------------------------
# Convolution via Unfolder / Folder (App. C)
# --------------------------------------------------------------------------
def conv_out_hw(H, W, kh, kw, stride, pad):
    return (H + 2 * pad - kh) // stride + 1, (W + 2 * pad - kw) // stride + 1


def unfold(x, kh, kw, stride, pad):
    """Unfolder: X [N, C, H, W] -> X_u [N*Ho*Wo, C*kh*kw].

    Row m = (n*Ho + oh)*Wo + ow, column k = (c*kh + i)*kw + j, value
    X[n, c, oh*stride - pad + i, ow*stride - pad + j] or 0 outside the image (R1).
    """
    x = np.asarray(x, dtype=f32)
    N, C, H, W = x.shape
    Ho, Wo = conv_out_hw(H, W, kh, kw, stride, pad)
    xp = np.zeros((N, C, H + 2 * pad, W + 2 * pad), dtype=f32)
    xp[:, :, pad:pad + H, pad:pad + W] = x
    cols = np.empty((N, Ho, Wo, C, kh, kw), dtype=f32)
    for i in range(kh):
        for j in range(kw):
            patch = xp[:, :, i:i + stride * (Ho - 1) + 1:stride, j:j + stride * (Wo - 1) + 1:stride]
            cols[:, :, :, :, i, j] = patch.transpose(0, 2, 3, 1)
    return cols.reshape(N * Ho * Wo, C * kh * kw)


def fold_int(acc_u, N, C, H, W, kh, kw, stride, pad):
    """Folder on integers: sum each unfolded entry back onto its input pixel.

    acc_u [N*Ho*Wo, C*kh*kw] int -> [N, C, H, W] int64; taps that fall in the
    padding are dropped.
    """
    Ho, Wo = conv_out_hw(H, W, kh, kw, stride, pad)
    a = np.asarray(acc_u, dtype=np.int64).reshape(N, Ho, Wo, C, kh, kw)
    out = np.zeros((N, C, H + 2 * pad, W + 2 * pad), dtype=np.int64)
    for i in range(kh):
        for j in range(kw):
            out[:, :, i:i + stride * (Ho - 1) + 1:stride, j:j + stride * (Wo - 1) + 1:stride] += \
                a[:, :, :, :, i, j].transpose(0, 3, 1, 2)
    return out[:, :, pad:pad + H, pad:pad + W]


def pixel_signs(x):
    """Pixel-major signs of x [N, C, H, W]: row p = (n H + h) W + w is sign(x[n, :, h, w]).
    The operand layout of the implicit convolution product below."""
    x = np.asarray(x, dtype=f32)
    N, C, H, W = x.shape
    return sign(x.transpose(0, 2, 3, 1).reshape(N * H * W, C))


def tap_major_signs(w):
    """Signs of w [D, C, kh, kw] with the contraction index k' = t C + c of tap t = i kw + j."""
    w = np.asarray(w, dtype=f32)
    D, C, kh, kw = w.shape
    return sign(w.transpose(0, 2, 3, 1).reshape(D, kh * kw * C))


def implicit_conv_acc(x, w, pad):
    """Binary product of a stride-1 convolution with the Unfolder of App. C left implicit:
    acc[(n Ho + oh) Wo + ow, d] = sum over taps (i, j), then channels c, of
    sign(x)[n, c, oh + i - pad, ow + j - pad] sign(w)[d, c, i, j], where a tap in the
    zero padding has sign -1 (R1).  Exact int64."""
    x = np.asarray(x, dtype=f32)
    N, C, H, W = x.shape
    D, _, kh, kw = np.asarray(w).shape
    Ho, Wo = conv_out_hw(H, W, kh, kw, 1, pad)
    sx = np.full((N, C, H + 2 * pad, W + 2 * pad), -1, dtype=np.int64)
    sx[:, :, pad:pad + H, pad:pad + W] = sign(x)
    sw = sign(w).astype(np.int64)
    acc = np.zeros((N, Ho, Wo, D), dtype=np.int64)
    for i in range(kh):
        for j in range(kw):
            acc += np.einsum("nchw,dc->nhwd", sx[:, :, i:i + Ho, j:j + Wo], sw[:, :, i, j])
    return acc.reshape(N * Ho * Wo, D)


# --------------------------------------------------------------------------
# Backward, step 1: group ranges (Sec. 3.2, PSQ Sec. 5.2, PCQ Sec. 5.3)
# --------------------------------------------------------------------------
def grad_to_quantize(gy, gamma):
    """G = gY (.) Gamma (reading R2); gamma None means G = gY."""
    gy = np.asarray(gy, dtype=f32)
    if gamma is None:
        return gy.copy()
    return (gy * np.asarray(gamma, dtype=f32)[None, :]).astype(f32)


def sample_ranges(g, rows_per_group):
    """Per-sample-group zero point Z = min and range R = max - min (fp32)."""
    M, D = g.shape
    assert M % rows_per_group == 0
    grp = g.reshape(M // rows_per_group, rows_per_group * D)
    z = grp.min(axis=1).astype(f32)
    r = (grp.max(axis=1).astype(f32) - z).astype(f32)
    return z, r


def channel_ranges(g):
    """Per-channel (column) zero point and range (fp32)."""
    z = g.min(axis=0).astype(f32)
    r = (g.max(axis=0).astype(f32) - z).astype(f32)
    return z, r


# --------------------------------------------------------------------------
# Backward, step 2: AGP keep probabilities and masks (Sec. 5.2)
# --------------------------------------------------------------------------
def fixed_point_ranges(r):
    """R~_i = floor(R_i 2^(40 - E)) with 2^(E-1) <= max R < 2^E (exact)."""
    r = np.asarray(r, dtype=f32)
    rmax = float(r.max()) if r.size else 0.0
    if rmax <= 0.0:
        return [0] * r.size
    _, e = np.frexp(rmax)
    return [int(np.floor(np.ldexp(float(v), FIXED_POINT_BITS - int(e)))) for v in r]


def kept_capacity(n, bits, mode):
    """Upper bound on the number of kept groups."""
    if bits == 1 or mode == BERNOULLI:
        return n
    return -(-n // bits)


def agp_probabilities(r, bits, mode=SYSTEMATIC):
    """Keep probabilities of Sec. 5.2 as integers P_i = floor(p_i 2^32).

    Reading R3 (water-filling): sort the fixed-point ranges descending (ties:
    lower index first); t* is the first t with (n - b t) R~_(t) <= b S_t,
    S_t = sum of the sorted ranges from position t on.  The t* largest groups
    get p = 1, the rest p_i = (n - b t*) R~_i / (b S_t*), so sum p = n/b and
    p is proportional to R among uncapped groups.  With b = 1 every group is
    kept.  TOPK (App. B) gives P = 2^32 to the floor(n/b) (at least 1) largest.
    Returns (P list of ints, order list = sorted group ids).
    """
    n = len(r)
    if bits == 1:
        return [TWO32] * n, list(range(n))
    rt = fixed_point_ranges(r)
    order = sorted(range(n), key=lambda i: (-rt[i], i))
    P = [0] * n
    if mode == TOPK:
        k = max(1, n // bits) if n else 0
        for i in order[:k]:
            P[i] = TWO32
        return P, order
    suffix = [0] * (n + 1)
    for t in range(n - 1, -1, -1):
        suffix[t] = suffix[t + 1] + rt[order[t]]
    tstar = n
    for t in range(n):
        if (n - bits * t) * rt[order[t]] <= bits * suffix[t]:
            tstar = t
            break
    for i in order[:tstar]:
        P[i] = TWO32
    s = suffix[tstar]
    if s > 0:
        num = n - bits * tstar
        for i in order[tstar:]:
            P[i] = min(TWO32, (num * rt[i] * TWO32) // (bits * s))
    return P, order


def agp_masks(P, seed, stream, mode=SYSTEMATIC):
    """Masks m_i with P(m_i = 1) = P_i 2^-32 (reading R4).  Returns bool [n]."""
    n = len(P)
    if mode == BERNOULLI:
        u = uniform_u32(seed, stream, np.arange(n, dtype=np.uint64)).astype(np.int64)
        return np.array([int(u[i]) < P[i] for i in range(n)], dtype=bool)
    if mode == TOPK:
        return np.array([p == TWO32 for p in P], dtype=bool)
    c = int(uniform_u32(seed, stream, np.uint64(0)))
    kept = np.zeros(n, dtype=bool)
    for i in range(n):
        kept[i] = ((c + P[i]) >> 32) > (c >> 32)
        c += P[i]
    return kept


def select_groups(r, bits, mode, seed, stream):
    """AGP selection of one grouping: kept ids (ascending) and p^ per group."""
    P, _ = agp_probabilities(r, bits, mode)
    if bits == 1:
        kept = np.ones(len(P), dtype=bool)
    else:
        kept = agp_masks(P, seed, stream, mode)
    p_hat = np.array([p / TWO32 for p in P], dtype=np.float64)
    return np.nonzero(kept)[0].astype(np.int64), p_hat, P


# --------------------------------------------------------------------------
# Backward, step 3: stochastic rounding to b-bit codes (Sec. 3.2, reading R5)
# --------------------------------------------------------------------------
def sr_codes(x, z, r, bits, seed, stream, flat_index):
    """Unbiased b-bit codes of x under zero point z and range r (fp32 ops).

    x, z, r broadcast together; flat_index gives the Philox word index of each
    element (its row-major position m*D + j in G = [M, D] for PSQ, its
    column-major position j*M + m for PCQ).
    """
    B = f32((1 << bits) - 1)
    x = np.asarray(x, dtype=f32)
    z = np.asarray(z, dtype=f32)
    r = np.asarray(r, dtype=f32)
    with np.errstate(divide="ignore", invalid="ignore", over="ignore"):
        inv = (B / r).astype(f32)
        t = ((x - z).astype(f32) * inv).astype(f32)
        fl = np.floor(t).astype(f32)
        frac = (t - fl).astype(f32)
    w = uniform_u32(seed, stream, flat_index)
    u = ((w >> np.uint32(8)).astype(np.float64) * 2.0 ** -24).astype(f32)
    q = fl + (u < frac).astype(f32)
    q = np.clip(q, f32(0), B)
    degenerate = ~((r > 0) & np.isfinite(inv))
    q = np.where(np.broadcast_to(degenerate, q.shape), f32(0), q)
    return q.astype(np.int64)


def group_scale(r, z, p_hat, bits):
    """S' = R / (B p^) and Z' = Z / p^ (float64 arithmetic, rounded to fp32)."""
    B = float((1 << bits) - 1)
    s = np.array([np.float64(rv) / (B * ph) for rv, ph in zip(np.asarray(r, np.float64), p_hat)],
                 dtype=np.float64).astype(f32)
    zz = np.array([np.float64(zv) / ph for zv, ph in zip(np.asarray(z, np.float64), p_hat)],
                  dtype=np.float64).astype(f32)
    return s, zz


def agp_quantize(g, group_axis, rows_per_group, bits, mode, seed):
    """AGP + per-group quantization of G along one grouping (Sec. 5.2 / 5.3).

    group_axis 0: sample groups of `rows_per_group` consecutive rows (PSQ);
    group_axis 1: channel groups = columns (PCQ).  Returns a dict with Z, R,
    P, p_hat, kept ids, per-kept scale / zero and the codes of the kept groups:
    PSQ codes [kept*rpg, D] (row-major, kept order), PCQ codes [kept, M].
    """
    M, D = g.shape
    if group_axis == 0:
        z, r = sample_ranges(g, rows_per_group)
        stream_sel, stream_sr = STREAM_SEL_SAMPLE, STREAM_SR_PSQ
    else:
        z, r = channel_ranges(g)
        stream_sel, stream_sr = STREAM_SEL_CHANNEL, STREAM_SR_PCQ
    kept, p_hat, P = select_groups(r, bits, mode, seed, stream_sel)
    scale, zero = group_scale(r[kept], z[kept], p_hat[kept], bits)
    if group_axis == 0:
        rows = (kept[:, None] * rows_per_group + np.arange(rows_per_group)[None, :]).reshape(-1)
        grp = np.repeat(kept, rows_per_group)
        flat = rows[:, None].astype(np.uint64) * np.uint64(D) + np.arange(D, dtype=np.uint64)[None, :]
        codes = sr_codes(g[rows, :], z[grp][:, None], r[grp][:, None], bits, seed, stream_sr, flat)
    else:
        flat = kept.astype(np.uint64)[:, None] * np.uint64(M) + np.arange(M, dtype=np.uint64)[None, :]
        codes = sr_codes(g[:, kept].T, z[kept][:, None], r[kept][:, None], bits, seed, stream_sr, flat)
    return dict(z=z, r=r, P=P, p_hat=p_hat, kept=kept, scale=scale, zero=zero, codes=codes,
                bits=bits, group_axis=group_axis, rows_per_group=rows_per_group)


def scq_quantize(g, rows_per_group, bits_s, mode_s, seed_s, bits_c, mode_c, seed_c):
    """SCQ (Sec. 5.3): PSQ branch for grad_input, PCQ branch for grad_weight."""
    return (agp_quantize(g, 0, rows_per_group, bits_s, mode_s, seed_s),
            agp_quantize(g, 1, 1, bits_c, mode_c, seed_c))


def bit_planes(codes, bits):
    """Lossless bit-plane decomposition x = sum_i 2^(i-1) x^i (Sec. 5.2)."""
    codes = np.asarray(codes, dtype=np.int64)
    return np.stack([(codes >> p) & 1 for p in range(bits)], axis=0).astype(np.int8)


# --------------------------------------------------------------------------
# Backward, step 4: the two integer GEMMs and SCQ dequantization (Eq. 21, Sec. 5.3)
# --------------------------------------------------------------------------
def dequant(scale, acc, zero, colsum):
    """out = S' * float(acc) + Z' * float(colsum), fp32 ops in that order (R6)."""
    a = (np.asarray(scale, f32) * np.asarray(acc).astype(f32)).astype(f32)
    c = (np.asarray(zero, f32) * np.asarray(colsum).astype(f32)).astype(f32)
    return (a + c).astype(f32)


def bwd_input(psq, w, M):
    """grad of the unfolded input: S_PSQ Q_PSQ sign(W) (per-sample side of SCQ).

    acc [kept*rpg, K] = codes @ sign(w); dX_u[m, k] = S'_g acc + Z'_g colsum_D(sign w)[k]
    for rows of kept groups, 0 for pruned rows.  Returns (acc, dx_u [M, K]).
    """
    sw = sign(w)
    acc = int_matmul(psq["codes"], sw.T)
    cs = sw.astype(np.int64).sum(axis=0)
    rpg = psq["rows_per_group"]
    K = sw.shape[1]
    dx = np.zeros((M, K), dtype=f32)
    for s, g in enumerate(psq["kept"]):
        rows = slice(g * rpg, (g + 1) * rpg)
        dx[rows] = dequant(psq["scale"][s], acc[s * rpg:(s + 1) * rpg], psq["zero"][s], cs[None, :])
    return acc, dx


def bwd_input_conv(psq, w, N, C, H, W, kh, kw, stride, pad):
    """Conv grad_input: fold the int32 accumulators first (exact), then dequantize.

    dX[n] = S'_n * float(fold(acc)[n]) + Z'_n * float(fold(colsum)) for kept
    samples n, 0 for pruned ones.  Returns (acc, acc_fold, cs_fold, dx).
    """
    Ho, Wo = conv_out_hw(H, W, kh, kw, stride, pad)
    rpg = Ho * Wo
    sw = sign(w.reshape(w.shape[0], -1))
    acc = int_matmul(psq["codes"], sw.T)
    cs = sw.astype(np.int64).sum(axis=0)
    full = np.zeros((N * rpg, C * kh * kw), dtype=np.int64)
    for s, g in enumerate(psq["kept"]):
        full[g * rpg:(g + 1) * rpg] = acc[s * rpg:(s + 1) * rpg]
    acc_fold = fold_int(full, N, C, H, W, kh, kw, stride, pad)
    cs_fold = fold_int(np.broadcast_to(cs[None, :], (rpg, cs.size)), 1, C, H, W, kh, kw, stride, pad)[0]
    dx = np.zeros((N, C, H, W), dtype=f32)
    for s, g in enumerate(psq["kept"]):
        dx[g] = dequant(psq["scale"][s], acc_fold[g], psq["zero"][s], cs_fold)
    return acc, acc_fold, cs_fold, dx


def bwd_weight(pcq, x_u, D):
    """grad of the weight: sign(X)^T Q_PCQ S_PCQ (per-channel side of SCQ).

    acc [kept, K] = codes^c @ sign(x_u); dW[j, k] = S^c'_j acc + Z^c'_j colsum_M(sign x_u)[k]
    for kept channels j, 0 for pruned channels.  Returns (acc, dw [D, K]).
    """
    sx = sign(x_u)
    acc = int_matmul(pcq["codes"], sx.T)
    cs = sx.astype(np.int64).sum(axis=0)
    dw = np.zeros((D, sx.shape[1]), dtype=f32)
    for s, j in enumerate(pcq["kept"]):
        dw[j] = dequant(pcq["scale"][s], acc[s], pcq["zero"][s], cs)
    return acc, dw


# --------------------------------------------------------------------------
# One whole layer step (App. C, Algorithm 1 without the weight update)
# --------------------------------------------------------------------------
def layer_step_linear(x, w, gamma, gy, bits_s, mode_s, seed_s, bits_c, mode_c, seed_c,
                      rows_per_group=1):
    """Forward + SCQ backward of a binarized fully connected layer."""
    acc_y, y = forward(x, w, gamma)
    g = grad_to_quantize(gy, gamma)
    psq, pcq = scq_quantize(g, rows_per_group, bits_s, mode_s, seed_s, bits_c, mode_c, seed_c)
    acc_dx, dx = bwd_input(psq, w, x.shape[0])
    acc_dw, dw = bwd_weight(pcq, x, w.shape[0])
    return dict(acc_y=acc_y, y=y, psq=psq, pcq=pcq, acc_dx=acc_dx, dx=dx, acc_dw=acc_dw, dw=dw)


def layer_step_conv(x, w, gamma, gy, stride, pad, bits_s, mode_s, seed_s, bits_c, mode_c, seed_c):
    """Forward + SCQ backward of a binarized convolution through Unfolder / Folder.

    x [N, C, H, W], w [D, C, kh, kw], gy [N*Ho*Wo, D] (NHWC rows, same layout as y).
    """
    N, C, H, W = x.shape
    D, _, kh, kw = w.shape
    x_u = unfold(x, kh, kw, stride, pad)
    w_u = w.reshape(D, -1)
    acc_y, y = forward(x_u, w_u, gamma)
    Ho, Wo = conv_out_hw(H, W, kh, kw, stride, pad)
    g = grad_to_quantize(gy, gamma)
    psq, pcq = scq_quantize(g, Ho * Wo, bits_s, mode_s, seed_s, bits_c, mode_c, seed_c)
    acc_dx, acc_fold, cs_fold, dx = bwd_input_conv(psq, w, N, C, H, W, kh, kw, stride, pad)
    acc_dw, dw = bwd_weight(pcq, x_u, D)
    return dict(x_u=x_u, acc_y=acc_y, y=y, psq=psq, pcq=pcq, acc_dx=acc_dx, acc_fold=acc_fold,
                cs_fold=cs_fold, dx=dx, acc_dw=acc_dw, dw=dw.reshape(w.shape))
