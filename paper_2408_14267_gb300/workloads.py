"""Seeded synthetic layer workloads (shapes and value distributions only).

This module holds none of the method's arithmetic: it only draws inputs.  Both
the CUDA path and the CPU oracle are fed from here.  Shapes follow the layers
of the networks the paper trains (VGG-16 and ResNet-18 on 32x32 and 224x224
images, App. D); value distributions mimic the heterogeneous per-sample
gradient ranges that motivate AGP (Sec. 5.2, Fig. "dis").  No dataset is used.

A workload is a dict:
  kind 'linear': x [M, K], w [D, K]
  kind 'conv'  : x [N, C, H, W], w [D, C, kh, kw], stride, pad
plus gamma [D] (the learnable Gamma of Sec. 5.1, initialised to
mean|X| * mean|W|), gy [M, D] (rows = samples, or NHWC pixels for conv),
and the AGP settings of the two SCQ branches.
"""
import numpy as np

SYSTEMATIC, BERNOULLI, TOPK = 0, 1, 2


def _gamma(x, w, D):
    g = np.float32(np.abs(x).astype(np.float64).mean() * np.abs(w).astype(np.float64).mean())
    return np.full(D, g, dtype=np.float32)


def _agp(bits_s, bits_c, seed, mode=SYSTEMATIC):
    return dict(bits_s=bits_s, mode_s=mode, seed_s=seed, bits_c=bits_c, mode_c=mode, seed_c=seed + 1)


def linear_small(seed=1000, qseed=0xF071):
    """Single linear layer, batch 64, 512 -> 512, 2-bit kept groups, keep 1/2."""
    rng = np.random.default_rng(seed)
    M, K, D = 64, 512, 512
    x = rng.standard_normal((M, K), dtype=np.float32)
    w = (0.02 * rng.standard_normal((D, K))).astype(np.float32)
    s = 10.0 ** rng.uniform(-2, 2, size=(M, 1))
    gy = (rng.laplace(0.0, 1e-3, size=(M, D)) * s).astype(np.float32)
    return dict(name="linear 64x512x512 b2", kind="linear", x=x, w=w, gamma=_gamma(x, w, D), gy=gy,
                rows_per_group=1, **_agp(2, 2, qseed))


def conv_layer(name, N, C, H, W, D, k, stride, pad, bits, seed, qseed, x_dist="normal",
               gy_dist="normal", gy_scale=1e-3, sample_sigma=None):
    """One convolution layer of the given shape with seeded inputs."""
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((N, C, H, W), dtype=np.float32)
    if x_dist == "absnormal":
        x = np.abs(x)
    elif x_dist == "relu":
        x = np.maximum(x, 0)
    fan_in = C * k * k
    w = (np.sqrt(2.0 / fan_in) * rng.standard_normal((D, C, k, k))).astype(np.float32)
    Ho = (H + 2 * pad - k) // stride + 1
    Wo = (W + 2 * pad - k) // stride + 1
    M = N * Ho * Wo
    if gy_dist == "t3":
        g = rng.standard_t(3, size=(M, D))
    else:
        g = rng.standard_normal((M, D))
    g = g * gy_scale
    if sample_sigma is not None:
        s = np.exp(sample_sigma * rng.standard_normal((N, 1, 1)))
        g = (g.reshape(N, Ho * Wo, D) * s).reshape(M, D)
    return dict(name=name, kind="conv", x=x, w=w, stride=stride, pad=pad, gamma=_gamma(x, w, D),
                gy=g.astype(np.float32), rows_per_group=Ho * Wo, **_agp(bits, bits, qseed))


def resnet18_cifar_conv(seed=1001, qseed=0xF072):
    """ResNet-18 (CIFAR) 3x3 conv 256 -> 256 on 8x8 maps, batch 128, b = 4, keep 1/4.

    X post-ReLU |N(0,1)|, W ~ N(0, 2/2304), gY Student-t(3) scaled 1e-3.
    Unfolded: M = 8192, K = 2304, D = 256.
    """
    return conv_layer("resnet18-cifar conv3x3 256->256 8x8 b128", 128, 256, 8, 8, 256, 3, 1, 1, 4,
                      seed, qseed, x_dist="absnormal", gy_dist="t3")


# VGG-16 on 32x32 inputs, batch 128: (C_in, C_out, H) of the 13 convs.
VGG16_CONVS = [(3, 64, 32), (64, 64, 32), (64, 128, 16), (128, 128, 16), (128, 256, 8), (256, 256, 8),
               (256, 256, 8), (256, 512, 4), (512, 512, 4), (512, 512, 4), (512, 512, 2), (512, 512, 2),
               (512, 512, 2)]
VGG16_FCS = [(512, 512), (512, 512), (512, 10)]

# ResNet-18 on 224x224 inputs, batch 64: (name, C_in, C_out, H_in, k, stride, pad).
RESNET18_IMAGENET = [("stem", 3, 64, 224, 7, 2, 3)] + \
    [("layer1", 64, 64, 56, 3, 1, 1)] + \
    [("layer2.conv1", 64, 128, 56, 3, 2, 1), ("layer2.down", 64, 128, 56, 1, 2, 0),
     ("layer2.conv", 128, 128, 28, 3, 1, 1)] + \
    [("layer3.conv1", 128, 256, 28, 3, 2, 1), ("layer3.down", 128, 256, 28, 1, 2, 0),
     ("layer3.conv", 256, 256, 14, 3, 1, 1)] + \
    [("layer4.conv1", 256, 512, 14, 3, 2, 1), ("layer4.down", 256, 512, 14, 1, 2, 0),
     ("layer4.conv", 512, 512, 7, 3, 1, 1)]


def vgg16_layers(bits=4, seed=1002, qseed=0xF073):
    """The 13 convs + 3 FCs of VGG-16 (CIFAR, batch 128); per-sample log-normal(2) gY."""
    out = []
    for i, (c, d, h) in enumerate(VGG16_CONVS):
        out.append(conv_layer(f"vgg16.conv{i + 1} {c}->{d} {h}x{h}", 128, c, h, h, d, 3, 1, 1, bits,
                              seed + 17 * i, qseed + i, sample_sigma=2.0))
    for i, (k, d) in enumerate(VGG16_FCS):
        rng = np.random.default_rng(seed + 1000 + i)
        x = rng.standard_normal((128, k), dtype=np.float32)
        w = (np.sqrt(2.0 / k) * rng.standard_normal((d, k))).astype(np.float32)
        gy = (1e-3 * rng.standard_normal((128, d)) * np.exp(2.0 * rng.standard_normal((128, 1)))).astype(np.float32)
        out.append(dict(name=f"vgg16.fc{i + 1} {k}->{d}", kind="linear", x=x, w=w, gamma=_gamma(x, w, d), gy=gy,
                        rows_per_group=1, **_agp(bits, bits, qseed + 100 + i)))
    return out


def resnet18_imagenet_layers(seed=1003, qseed=0xF074):
    """Every distinct conv shape of ResNet-18 at 224x224, batch 64, b = 4, keep 1/4."""
    return [conv_layer(f"resnet18.{n} {c}->{d} {h}x{h} k{k}s{s}", 64, c, h, h, d, k, s, p, 4, seed + 31 * i,
                       qseed + i) for i, (n, c, d, h, k, s, p) in enumerate(RESNET18_IMAGENET)]


def sweep_point(M, K, D, groups, bits, seed=1004, qseed=0xF075):
    """GEMM-shaped layer for the throughput sweep: groups of M/groups rows."""
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((M, K), dtype=np.float32)
    w = rng.standard_normal((D, K), dtype=np.float32)
    s = 10.0 ** rng.uniform(-2, 2, size=(groups, 1, 1))
    gy = (rng.laplace(0.0, 1e-3, size=(groups, M // groups, D)) * s).reshape(M, D).astype(np.float32)
    return dict(name=f"sweep M{M} K{K} D{D} G{groups} b{bits}", kind="linear", x=x, w=w,
                gamma=np.ones(D, dtype=np.float32), gy=gy, rows_per_group=M // groups, **_agp(bits, bits, qseed))


def sweep_point_device(M, K, D, groups, bits, device, seed=1004, qseed=0xF075):
    """The sweep recipe of `sweep_point`, drawn on the device with torch's generator (the large
    points do not fit a host draw in reasonable time): X, W ~ N(0,1), gY = Laplace(0, 1e-3) x
    10^U(-2,2) per group of M/groups rows, Gamma = 1.  Timing only: parity tests draw their
    sweep points with `sweep_point` so that the oracle sees the same numbers."""
    import torch
    g = torch.Generator(device=device).manual_seed(seed)
    x = torch.randn(M, K, generator=g, device=device)
    w = torch.randn(D, K, generator=g, device=device)
    # u strictly inside (-1/2, 1/2): rand() can return 0, and u = -1/2 would give -inf
    u = torch.rand(M, D, generator=g, device=device) + (0.5 * 2.0 ** -24 - 0.5)
    lap = -1e-3 * torch.sign(u) * torch.log1p(-2.0 * u.abs())
    s = 10.0 ** (torch.rand(groups, 1, 1, generator=g, device=device) * 4.0 - 2.0)
    gy = (lap.view(groups, M // groups, D) * s).view(M, D).contiguous()
    return dict(name=f"sweep M{M} K{K} D{D} G{groups} b{bits}", kind="linear", x=x, w=w,
                gamma=torch.ones(D, device=device), gy=gy, rows_per_group=M // groups, **_agp(bits, bits, qseed))

