"""The C-ABI library: it loads, exports every declared entry point, and rejects bad
arguments on the host before any launch (no GPU needed)."""
import ctypes as C
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2408_14267_gb300 import build, fqt1
    build.build()
    return fqt1.lib()


def declared_functions():
    names = []
    for h in os.listdir(os.path.join(ROOT, "include")):
        if h.endswith(".h"):
            txt = open(os.path.join(ROOT, "include", h)).read()
            names += re.findall(r"^\s*(?:[\w\s\*]+?)\b(fqt1_\w+)\s*\(", txt, flags=re.M)
    return sorted(set(names))


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert len(names) >= 13
    for n in names:
        assert hasattr(lib, n), n
    from paper_2408_14267_gb300 import fqt1
    assert sorted(fqt1.exported_names()) == names


def test_helpers(lib):
    from paper_2408_14267_gb300 import fqt1
    assert fqt1.packed_words(1) == 4 and fqt1.packed_words(128) == 4 and fqt1.packed_words(129) == 8
    assert fqt1.kept_capacity(64, 2, 0) == 32 and fqt1.kept_capacity(10, 4, 0) == 3
    assert fqt1.kept_capacity(10, 4, 1) == 10 and fqt1.kept_capacity(10, 1, 0) == 10
    assert fqt1.codes_ld(1) == 16 and fqt1.codes_ld(32) == 32 and fqt1.codes_ld(33) == 48


def test_argument_validation_without_launch(lib):
    """Every rejected call returns its status before touching the device."""
    from paper_2408_14267_gb300 import fqt1
    fake = C.c_void_p(0x10000)       # never dereferenced: validation fails first
    odd = C.c_void_p(0x10004)
    s = C.c_void_p(0)
    assert lib.fqt1_binarize_pack(None, 4, 4, 4, fake, None, None, s) == 1
    assert lib.fqt1_binarize_pack(fake, 4, 4, 3, fake, None, None, s) == 1          # ld < cols
    assert lib.fqt1_binarize_pack(fake, 4, 4, 4, None, None, None, s) == 1          # no output
    assert lib.fqt1_binarize_pack(odd, 4, 4, 4, fake, None, None, s) == 2           # misaligned
    assert lib.fqt1_im2col(fake, 1, 1, 2, 2, 5, 5, 1, 0, fake, None, None, s) == 1  # kernel larger than image
    assert lib.fqt1_fwd_gemm(fake, fake, 0, 4, 4, fake, None, fake, s) == 1
    assert lib.fqt1_fwd_gemm(fake, fake, 4, 4, 4, None, None, fake, s) == 1          # y without gamma
    bad_bits = fqt1.AgpParams(3, 0, 1, 1)
    ok = fqt1.AgpParams(2, 0, 1, 1)
    q = fqt1.QGrad(*(0x10000 for _ in range(9)), 64)
    st = fake
    assert lib.fqt1_agp_quantize_grad(fake, 8, 8, 0, None, C.byref(bad_bits), C.byref(q), fake, 4096, st, s) == 1
    assert lib.fqt1_agp_quantize_grad(fake, 8, 8, 2, None, C.byref(ok), C.byref(q), fake, 4096, st, s) == 1
    assert lib.fqt1_agp_quantize_grad(fake, 8, 8, 0, None, C.byref(ok), C.byref(q), fake, 4, st, s) == 4
    rpg3 = fqt1.AgpParams(2, 0, 1, 3)                                                  # 3 does not divide 8
    assert lib.fqt1_agp_quantize_grad(fake, 8, 8, 0, None, C.byref(rpg3), C.byref(q), fake, 4096, st, s) == 1
    bad_mode = fqt1.AgpParams(2, 7, 1, 1)
    assert lib.fqt1_scq_quantize(fake, 8, 8, None, C.byref(ok), C.byref(bad_mode), C.byref(q), C.byref(q), fake,
                                 4096, st, s) == 1
    big = fqt1.AgpParams(2, 0, 1, 1)
    qbig = fqt1.QGrad(*(0x10000 for _ in range(9)), 1 << 16)
    assert lib.fqt1_agp_quantize_grad(fake, 20000, 16, 0, None, C.byref(big), C.byref(qbig), fake, 1 << 20, st,
                                      s) == 3                                          # > 16384 groups
    assert lib.fqt1_bwd_input_gemm(C.byref(q), fake, fake, 8, 8, 8, C.byref(bad_bits), fake, fake, s) == 1
    assert lib.fqt1_bwd_weight_gemm(C.byref(q), fake, fake, 8, 8, 8, C.byref(ok), None, fake, None, 0, s) == 1
    assert lib.fqt1_col2im(fake, C.byref(q), fake, 1, 1, 4, 4, 3, 3, 0, 1, fake, s) == 1  # stride 0
