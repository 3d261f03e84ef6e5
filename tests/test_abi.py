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
    assert lib.fqt1_bwd_input_gemm(C.byref(q), fake, fake, 8, 8, 8, C.byref(bad_bits), fake, fake, s) == 1  # b = 3
    assert lib.fqt1_bwd_weight_gemm(C.byref(q), fake, fake, 8, 8, 8, C.byref(ok), None, fake, None, 0, s) == 1  # no acc
    assert lib.fqt1_col2im(fake, C.byref(q), fake, 1, 1, 4, 4, 3, 3, 0, 1, fake, s) == 1  # stride 0
    # column-major grad_input: ld below the kept rows (capacity 4 of 8 groups, 1 row each) or
    # not a multiple of 4; the Folder: stride 0, ld below Ho Wo, ld not a multiple of 4, and
    # an unaligned accumulator pointer
    assert lib.fqt1_bwd_input_gemm_colmajor(C.byref(q), fake, 8, 8, 8, C.byref(ok), fake, 32, 2, s) == 1
    assert lib.fqt1_bwd_input_gemm_colmajor(C.byref(q), fake, 8, 8, 8, C.byref(ok), fake, 32, 6, s) == 1
    assert lib.fqt1_bwd_input_gemm_colmajor(C.byref(q), fake, 8, 8, 8, C.byref(bad_bits), fake, 32, 8, s) == 1
    assert lib.fqt1_bwd_input_gemm_colmajor(C.byref(q), fake, 8, 8, 8, C.byref(ok), fake, 8, 8, s) == 1  # width 8
    assert lib.fqt1_bwd_input_gemm_colmajor(C.byref(q), fake, 8, 8, 8, C.byref(ok), fake, 16, 4, s) == 1  # ld % 8
    # int16 cannot hold the sums: 15 * 4096 and 15 * 2185 = 32775 > 32767 (the first width past
    # the bound, the binding's rule agreeing); q_wide's codes rows have room for D = 4096, so the
    # int16 bound is the only check these calls fail
    big_d = fqt1.AgpParams(4, 0, 1, 1)
    q_wide = fqt1.QGrad(*(0x10000 for _ in range(9)), 4096)
    assert lib.fqt1_bwd_input_gemm_colmajor(C.byref(q_wide), fake, 8, 4096, 8, C.byref(big_d), fake, 16, 8, s) == 1
    assert lib.fqt1_bwd_input_gemm_colmajor(C.byref(q_wide), fake, 8, 2185, 8, C.byref(big_d), fake, 16, 8, s) == 1
    assert fqt1.colmajor_acc_bits(4, 2185) == 32 and fqt1.colmajor_acc_bits(4, 2184) == 16
    # sign(W)^T rows of 8 bytes, below codes_ld(D = 8) = 16; no sign(W)^T at all
    assert lib.fqt1_bwd_input_gemm_colmajor_e4m3w(C.byref(q), fake, 8, 8, 8, 8, C.byref(ok), fake, 32, 8, s) == 1
    assert lib.fqt1_bwd_input_gemm_colmajor_e4m3w(C.byref(q), None, 16, 8, 8, 8, C.byref(ok), fake, 32, 8, s) == 1
    assert lib.fqt1_col2im_colmajor(fake, 32, 16, C.byref(q), fake, 1, 1, 4, 4, 3, 3, 0, 1, fake, s) == 1
    assert lib.fqt1_col2im_colmajor(fake, 32, 12, C.byref(q), fake, 1, 1, 4, 4, 3, 3, 1, 1, fake, s) == 1
    assert lib.fqt1_col2im_colmajor(fake, 32, 18, C.byref(q), fake, 1, 1, 4, 4, 3, 3, 1, 1, fake, s) == 1
    assert lib.fqt1_col2im_colmajor(fake, 16, 20, C.byref(q), fake, 1, 1, 4, 4, 3, 3, 1, 1, fake, s) == 1
    assert lib.fqt1_col2im_colmajor(fake, 24, 16, C.byref(q), fake, 1, 1, 4, 4, 3, 3, 1, 1, fake, s) == 1
    assert lib.fqt1_col2im_colmajor(C.c_void_p(0x10004), 32, 16, C.byref(q), fake, 1, 1, 4, 4, 3, 3, 1, 1, fake,
                                    s) == 2
    # C kh kw = 2^19 x 64 x 64 = 2^31 columns (C H W = 2^29): refused before any launch
    assert lib.fqt1_col2im_colmajor(fake, 32, 4, C.byref(q), fake, 1, 1 << 19, 32, 32, 64, 64, 1, 16, fake, s) == 3
    # shapes whose 32-bit index arithmetic would overflow are refused before any launch:
    # H + 2 pad >= 2^31, or Ho Wo >= 2^31 (a 1 x 1 input padded by 30000: 60001^2 outputs)
    huge, wide = 1 << 30, 30000
    p8 = fqt1.AgpParams(2, 0, 1, 1)
    for pad in (huge, wide):
        assert lib.fqt1_col2im_colmajor(fake, 32, 4, C.byref(q), fake, 1, 1, 1, 1, 1, 1, 1, pad, fake, s) == 3
        assert lib.fqt1_col2im(fake, C.byref(q), fake, 1, 1, 1, 1, 1, 1, 1, pad, fake, s) == 3
        assert lib.fqt1_bwd_input_fold(C.byref(q), fake, fake, 1, 1, 1, 1, 1, 1, 1, pad, C.c_int64(8), C.byref(p8),
                                       fake, s) == 3
        assert lib.fqt1_im2col(fake, 1, 1, 1, 1, 1, 1, 1, pad, fake, None, None, s) == 3
        assert lib.fqt1_im2col_path(1, 1, 1, 1, 1, 1, 1, pad) == -1


def test_implicit_conv_support_rules(lib):
    """Shapes the implicit-GEMM forward accepts: stride-1 "same" kernels, C a multiple of 128,
    and 128-pixel tiles of whole images or whole image rows (host logic, no GPU)."""
    ok = lambda *a: bool(lib.fqt1_conv_implicit_supported(*a))  # N, C, H, W, kh, kw, stride, pad
    assert ok(128, 256, 8, 8, 3, 3, 1, 1)           # whole images, 2 per tile
    assert ok(9, 128, 4, 4, 1, 1, 1, 0)             # 1x1, 8 images per tile
    assert ok(2, 128, 16, 16, 3, 3, 1, 1)           # 8 rows of 16 per tile
    assert ok(1, 512, 32, 32, 5, 5, 1, 2)           # 4 rows of 32, 5x5
    assert ok(64, 128, 2, 2, 3, 3, 1, 1)            # 32 images per tile
    assert not ok(2, 96, 8, 8, 3, 3, 1, 1)          # C not a multiple of 128
    assert not ok(2, 128, 8, 8, 3, 3, 2, 1)         # stride 2
    assert not ok(2, 128, 8, 8, 3, 3, 1, 0)         # not "same"
    assert not ok(2, 128, 8, 8, 3, 1, 1, 1)         # kh != kw
    assert not ok(2, 128, 12, 12, 3, 3, 1, 1)       # 144 pixels, rows of 12 do not tile 128
    assert not ok(2, 128, 12, 16, 3, 3, 1, 1)       # 8 rows per tile do not divide 12
    assert not ok(2, 128, 3, 3, 3, 3, 1, 1)         # 9 pixels do not divide 128


def test_unfolder_source_choice(lib):
    """Which Unfolder input a layer gives a contiguous x (host logic, no GPU): whole-image tiles
    (path 2) and pointwise windows (path 3) read x; region tiles (path 1) read sign planes packed
    first."""
    from paper_2408_14267_gb300 import fqt1
    assert fqt1.im2col_path(128, 256, 8, 8, 3, 3, 1, 1) == 2 and not fqt1.unfold_from_planes(128, 256, 8, 8, 3, 3, 1, 1)
    assert fqt1.im2col_path(64, 64, 56, 56, 1, 1, 2, 0) == 3 and not fqt1.unfold_from_planes(64, 64, 56, 56, 1, 1, 2, 0)
    for shape in [(128, 512, 4, 4, 3, 3, 1, 1), (16, 64, 2, 4, 3, 3, 1, 1), (128, 512, 2, 2, 3, 3, 1, 1),
                  (64, 512, 7, 7, 3, 3, 1, 1), (64, 256, 14, 14, 3, 3, 1, 1), (64, 3, 224, 224, 7, 7, 2, 3),
                  (8, 16, 1, 1, 3, 3, 1, 1)]:
        assert fqt1.im2col_path(*shape) == 1 and fqt1.unfold_from_planes(*shape), shape


def test_implicit_conv_validation_without_launch(lib):
    fake = C.c_void_p(0x10000)
    odd = C.c_void_p(0x10004)
    s = C.c_void_p(0)
    assert lib.fqt1_pack_pixels(fake, 2, 96, 8, 8, fake, s) == 3                   # C % 128
    assert lib.fqt1_pack_pixels(fake, 2, 128, 8, 8, odd, s) == 2                   # misaligned output
    assert lib.fqt1_pack_pixels(None, 2, 128, 8, 8, fake, s) == 1
    assert lib.fqt1_pack_weight_taps(fake, 4, 48, 3, 3, fake, s) == 3              # C % 32
    assert lib.fqt1_pack_weight_taps(fake, 0, 64, 3, 3, fake, s) == 1
    args = [fake, fake, 2, 128, 8, 8, 3, 3, 2, 1, C.c_int64(16), fake, None, None, fake, s]
    assert lib.fqt1_conv_fwd_implicit(*args) == 3                                  # stride 2
    args[8] = 1
    args[11] = None
    assert lib.fqt1_conv_fwd_implicit(*args) == 1                                  # no gamma
    args[11] = odd
    assert lib.fqt1_conv_fwd_implicit(*args) == 2                                  # misaligned gamma


def test_layout_and_e4m3_entry_points_validate_without_launch(lib):
    """Channels-last, e4m3 and workspace entry points reject bad arguments before any launch."""
    from paper_2408_14267_gb300 import fqt1
    fake = C.c_void_p(0x10000)
    odd = C.c_void_p(0x10004)
    s = C.c_void_p(0)
    # channels-last packing and the Unfolder from planes
    assert lib.fqt1_pack_planes_nhwc(fake, 2, 48, 8, 8, fake, s) == 3                     # C % 32
    assert lib.fqt1_pack_planes_nhwc(odd, 2, 64, 8, 8, fake, s) == 2                      # misaligned x
    assert lib.fqt1_pack_planes_nhwc(None, 2, 64, 8, 8, fake, s) == 1
    assert lib.fqt1_im2col_planes(None, 1, 32, 8, 8, 3, 3, 1, 1, fake, None, None, s) == 1
    assert lib.fqt1_im2col_planes(fake, 1, 32, 2, 2, 5, 5, 1, 0, fake, None, None, s) == 1  # kernel > image
    # e4m3 copies of the signs
    assert lib.fqt1_expand_signs_e4m3(fake, 4, 40, fake, C.c_int64(40), s) == 1            # ld % 16
    assert lib.fqt1_expand_signs_e4m3(fake, 4, 40, fake, C.c_int64(32), s) == 1            # ld < n
    assert lib.fqt1_expand_signs_e4m3(fake, 4, 40, odd, C.c_int64(48), s) == 2
    assert lib.fqt1_binarize_pack_e4m3(fake, 4, 40, 40, None, None, None, fake, C.c_int64(40), None, C.c_int64(0),
                                       s) == 1                                                  # ld_re % 16
    assert lib.fqt1_binarize_pack_e4m3(fake, 4, 40, 40, None, None, None, None, C.c_int64(0), None, C.c_int64(0),
                                       s) == 1                                                  # no output
    assert lib.fqt1_fwd_gemm_e4m3w(fake, fake, C.c_int64(32), 8, 8, 40, fake, None, None, fake, s) == 1  # ld < K
    assert lib.fqt1_fwd_gemm_e4m3w(fake, fake, C.c_int64(48), 8, 8, 40, None, None, None, fake, s) == 1  # gamma
    # channels-last Folders
    q = fqt1.QGrad(*(0x10000 for _ in range(9)), 64)
    p_ok = fqt1.AgpParams(4, 0, 1, 64)
    assert lib.fqt1_col2im_nhwc(None, C.byref(q), fake, 2, 8, 8, 8, 3, 3, 1, 1, fake, s) == 1
    assert lib.fqt1_bwd_input_fold_nhwc(C.byref(q), None, fake, 2, 8, 8, 8, 3, 3, 1, 1, C.c_int64(16), C.byref(p_ok),
                                        fake, s) == 1
    assert lib.fqt1_bwd_input_fold_e4m3w(C.byref(q), fake, C.c_int64(8), fake, 2, 8, 8, 8, 3, 3, 1, 1, C.c_int64(16),
                                         C.byref(p_ok), fake, s) == 1                           # ld_wt < D
    # workspace preparation
    assert lib.fqt1_scq_workspace_init(None, 64, s) == 1
    assert lib.fqt1_scq_workspace_init(fake, 0, s) == 1


_CTYPE_OF = {"int64_t": C.c_int64, "int32_t": C.c_int32, "size_t": C.c_size_t, "float": C.c_float,
             "uint64_t": C.c_uint64, "fqt1_status": C.c_int}


def _declarations():
    """(return type, name, [parameter types]) of every function declared in include/*.h."""
    out = []
    for h in sorted(os.listdir(os.path.join(ROOT, "include"))):
        if not h.endswith(".h"):
            continue
        txt = open(os.path.join(ROOT, "include", h)).read()
        txt = re.sub(r"/\*.*?\*/", " ", txt, flags=re.S)
        txt = re.sub(r"//[^\n]*", " ", txt)
        txt = re.sub(r"^\s*#[^\n]*", " ", txt, flags=re.M)
        for ret, name, params in re.findall(r"([\w\s\*]+?)\b(fqt1_\w+)\s*\(([^;{)]*)\)\s*;", txt):
            ret = " ".join(ret.strip().split("\n")[-1].split())
            ps = [" ".join(p.split()) for p in params.split(",")]
            ps = [] if ps == ["void"] or ps == [""] else ps
            types = [re.sub(r"\s*\b\w+$", "", p) if not p.endswith("*") else p for p in ps]
            out.append((ret, name, types))
    return out


def _expected_ctype(t):
    if "*" in t:
        return C.c_void_p
    t = t.replace("const ", "").strip()
    return _CTYPE_OF[t]


def test_binding_signatures_match_the_header():
    """Every ctypes signature in the binding has the header's arity and argument widths, so a
    wrong int32 / int64 / size_t or a missing argument fails here rather than on a GPU."""
    from paper_2408_14267_gb300 import fqt1
    decls = _declarations()
    assert {n for _, n, _ in decls} == set(fqt1._SIGS)
    for ret, name, types in decls:
        restype, argtypes = fqt1._SIGS[name]
        assert len(argtypes) == len(types), (name, types)
        for i, (t, a) in enumerate(zip(types, argtypes)):
            assert a is _expected_ctype(t), (name, i, t, a)
        want = C.c_char_p if ret == "const char*" else _expected_ctype(ret)
        assert restype is want, (name, ret, restype)
