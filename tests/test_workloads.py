"""The seeded input recipes: layer shapes of the networks the paper trains (App. D) and the
value distributions of the synthetic stand-ins (heterogeneous per-sample gradient ranges,
Sec. 5.2). No GPU; the large ResNet-18 tensors are not drawn, only their shapes computed."""
import numpy as np
import pytest

from paper_2408_14267_gb300 import workloads as wl


def _mkd(c, d, h, k, s, p, batch):
    ho = (h + 2 * p - k) // s + 1
    return batch * ho * ho, c * k * k, d


def test_vgg16_cifar_layer_shapes():
    """VGG-16 on 32x32, batch 128: 3x3 convs with pad 1, pooling after conv 2, 4, 7, 10, 13."""
    got = [_mkd(c, d, h, 3, 1, 1, 128) for c, d, h in wl.VGG16_CONVS]
    want = [(131072, 27, 64), (131072, 576, 64), (32768, 576, 128), (32768, 1152, 128),
            (8192, 1152, 256), (8192, 2304, 256), (8192, 2304, 256), (2048, 2304, 512),
            (2048, 4608, 512), (2048, 4608, 512), (512, 4608, 512), (512, 4608, 512), (512, 4608, 512)]
    assert got == want
    assert wl.VGG16_FCS == [(512, 512), (512, 512), (512, 10)]


def test_resnet18_imagenet_layer_shapes():
    """ResNet-18 on 224x224, batch 64: 7x7/2 stem, four stages of 3x3 convs, 1x1/2 downsamples."""
    got = {n: _mkd(c, d, h, k, s, p, 64) for n, c, d, h, k, s, p in wl.RESNET18_IMAGENET}
    assert got == {
        "stem": (802816, 147, 64), "layer1": (200704, 576, 64),
        "layer2.conv1": (50176, 576, 128), "layer2.down": (50176, 64, 128), "layer2.conv": (50176, 1152, 128),
        "layer3.conv1": (12544, 1152, 256), "layer3.down": (12544, 128, 256), "layer3.conv": (12544, 2304, 256),
        "layer4.conv1": (3136, 2304, 512), "layer4.down": (3136, 256, 512), "layer4.conv": (3136, 4608, 512)}


def test_bench_workload_recipe():
    """ResNet-18 CIFAR conv 256 -> 256 on 8x8, batch 128: X = abs(N(0,1)), W ~ N(0, 2/2304),
    gY = 1e-3 Student-t(3) (variance 3e-6), Gamma = mean abs(X) mean abs(W), b = 4 both branches."""
    w = wl.resnet18_cifar_conv()
    assert w["x"].shape == (128, 256, 8, 8) and w["w"].shape == (256, 256, 3, 3)
    assert w["gy"].shape == (8192, 256) and w["rows_per_group"] == 64
    assert (w["stride"], w["pad"], w["bits_s"], w["bits_c"]) == (1, 1, 4, 4)
    assert w["x"].min() >= 0 and abs(w["x"].mean() - np.sqrt(2 / np.pi)) < 0.01
    assert abs(w["w"].std() - np.sqrt(2 / 2304)) / np.sqrt(2 / 2304) < 0.01
    q = np.quantile(w["gy"], [0.25, 0.75]) / 1e-3  # quartiles of t(3): -/+ 0.7649
    assert np.allclose(q, [-0.7649, 0.7649], atol=0.01)
    assert np.all(w["gamma"] == np.float32(np.abs(w["x"]).astype(np.float64).mean()
                                           * np.abs(w["w"]).astype(np.float64).mean()))
    assert w["seed_s"] != w["seed_c"]


def test_linear_recipe_has_four_decades_of_sample_ranges():
    """Laplace(0, 1e-3) gradients scaled by 10^U(-2, 2) per sample: ranges spread over about
    four decades, the heterogeneity AGP exploits (Sec. 5.2)."""
    w = wl.linear_small()
    assert w["x"].shape == (64, 512) and w["w"].shape == (512, 512) and w["gy"].shape == (64, 512)
    r = w["gy"].max(axis=1) - w["gy"].min(axis=1)
    assert 2.5 < np.log10(r.max() / r.min()) < 4.5
    assert (w["bits_s"], w["bits_c"], w["rows_per_group"]) == (2, 2, 1)


def test_recipes_are_seeded():
    a, b = wl.linear_small(), wl.linear_small()
    for k in ("x", "w", "gy", "gamma"):
        assert np.array_equal(a[k], b[k])
    c = wl.linear_small(seed=7)
    assert not np.array_equal(a["x"], c["x"])


@pytest.mark.parametrize("groups", [64, 256])
def test_sweep_point_groups(groups):
    w = wl.sweep_point(1024, 1024, 1024, groups, 4)
    assert w["rows_per_group"] == 1024 // groups
    r = w["gy"].reshape(groups, -1).max(axis=1) - w["gy"].reshape(groups, -1).min(axis=1)
    assert np.log10(r.max() / r.min()) > 2.5
