"""The C-ABI library builds, loads and exports what include/gemmi.h declares (no GPU needed).

Only host-side logic runs here: argument validation happens before any device
access, so invalid calls return GEMMI_EINVAL and empty problems return OK
without touching a GPU.
"""
import ctypes
import os
import re

import pytest

import paper_2302_07594_gb300 as gm

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "gemmi.h")


@pytest.fixture(scope="module")
def L():
    gm.build()
    return gm.lib()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    names = re.findall(r"^\s*(?:const\s+)?[a-z_0-9]+\s*\*?\s*([a-z_0-9]+)\s*\(", text, flags=re.M)
    return sorted(set(n for n in names if n not in ("if", "while")))


def test_header_declares_the_core_calls():
    names = declared_functions()
    for core in ("gemm_i16", "gemm_i8", "gemm_i16_ex", "gemm_i8_ex", "gemmi_last_error"):
        assert core in names


def test_library_exports_every_declared_symbol(L):
    missing = [n for n in declared_functions() if not hasattr(L, n)]
    assert missing == []
    assert sorted(declared_functions()) == sorted(gm.EXPORTED)


def test_no_oracle_or_cpu_fallback_symbols(L):
    # the product library must not contain the oracle: no symbol it defines names it
    import shutil
    import subprocess
    if shutil.which("nm") is None:
        pytest.skip("nm is not installed")
    out = subprocess.run(["nm", "-D", "--defined-only", gm.LIB_PATH], capture_output=True, text=True,
                         check=True).stdout
    assert "gemm_i16" in out
    assert "oracle" not in out


def test_version(L):
    assert "sm_103a" in gm.version()


@pytest.mark.parametrize("args", [
    (-1, 4, 4, 4, 4, 4),    # negative m
    (4, 4, 4, 3, 4, 4),     # lda < k
    (4, 4, 4, 4, 3, 4),     # ldb < n
    (4, 4, 4, 4, 4, 3),     # ldc < n
])
def test_invalid_arguments(L, args):
    m, n, k, lda, ldb, ldc = args
    dummy = ctypes.c_void_p(0x1000)
    rc = L.gemm_i16(m, n, k, dummy, lda, ctypes.c_void_p(0x2000), ldb, ctypes.c_void_p(0x3000), ldc)
    assert rc == gm.EINVAL
    assert gm.last_error() != ""


def test_null_and_overlap_rejected(L):
    assert L.gemm_i16(4, 4, 4, None, 4, ctypes.c_void_p(0x2000), 4, ctypes.c_void_p(0x3000), 4) == gm.EINVAL
    assert L.gemm_i16(4, 4, 4, ctypes.c_void_p(0x1000), 4, ctypes.c_void_p(0x2000), 4, None, 4) == gm.EINVAL
    # C overlapping A
    assert L.gemm_i16(4, 4, 4, ctypes.c_void_p(0x1000), 4, ctypes.c_void_p(0x90000), 4,
                      ctypes.c_void_p(0x1008), 4) == gm.EINVAL
    assert "overlap" in gm.last_error()


def test_leading_dimension_overflow_rejected(L):
    """An operand whose extent ((rows - 1) * ld + cols elements) overflows 64 bits is refused, not
    wrapped around into a span that could slip past the overlap check."""
    huge = 1 << 62
    a, b, c = ctypes.c_void_p(0x1000), ctypes.c_void_p(0x2000), ctypes.c_void_p(0x3000)
    assert L.gemm_i16(4, 4, 4, a, huge, b, 4, c, 4) == gm.EINVAL
    assert "overflow" in gm.last_error()
    assert L.gemm_i8(4, 4, 4, a, 4, b, huge, c, 4) == gm.EINVAL
    assert L.gemm_i16_noalloc(4, 4, 4, a, 4, b, 4, c, huge, None) == gm.EINVAL
    assert "overflow" in gm.last_error()


def test_read_probe_argument_checks(L):
    L.gemmi_stream_read_probe.argtypes = [ctypes.c_int64, ctypes.c_int64, ctypes.c_void_p, ctypes.c_int64,
                                          ctypes.c_void_p]
    assert L.gemmi_stream_read_probe(64, 64, ctypes.c_void_p(0x1008), 64, None) == gm.EINVAL  # not 16-byte aligned
    assert L.gemmi_stream_read_probe(64, 64, ctypes.c_void_p(0x1000), 60, None) == gm.EINVAL  # ldb < n
    assert L.gemmi_stream_read_probe(64, 60, ctypes.c_void_p(0x1000), 60, None) == gm.EINVAL  # ldb % 8 != 0
    assert L.gemmi_stream_read_probe(0, 64, None, 64, None) == gm.OK


def test_empty_problems_are_noops(L):
    assert L.gemm_i16(0, 4, 4, None, 4, None, 4, None, 4) == gm.OK
    assert L.gemm_i8(4, 0, 4, None, 4, None, 1, None, 1) == gm.OK
    # k == 0: C untouched, A and B may be null
    assert L.gemm_i16(3, 3, 0, None, 1, None, 3, ctypes.c_void_p(0x3000), 3) == gm.OK


def test_i4_argument_checks(L):
    """gemm_i4 counts lda and ldb in packed bytes: ceil(k/2) and ceil(n/2) are the minimums."""
    a, b, c = ctypes.c_void_p(0x1000), ctypes.c_void_p(0x90000), ctypes.c_void_p(0x200000)
    assert L.gemm_i4(4, 5, 7, a, 3, b, 3, c, 5) == gm.EINVAL       # lda < ceil(7/2) = 4
    assert "lda" in gm.last_error()
    assert L.gemm_i4(4, 5, 7, a, 4, b, 2, c, 5) == gm.EINVAL       # ldb < ceil(5/2) = 3
    assert "ldb" in gm.last_error()
    assert L.gemm_i4(4, 5, 7, a, 4, b, 3, c, 4) == gm.EINVAL       # ldc < n
    assert L.gemm_i4(-1, 5, 7, a, 4, b, 3, c, 5) == gm.EINVAL
    assert L.gemm_i4(4, 5, 7, None, 4, b, 3, c, 5) == gm.EINVAL
    assert L.gemm_i4(4, 5, 7, a, 4, b, 3, ctypes.c_void_p(0x1002), 5) == gm.EINVAL  # C overlaps A
    assert "overlap" in gm.last_error()
    # empty problems and k == 0 are no-ops that touch no device
    assert L.gemm_i4(0, 5, 7, None, 4, None, 3, None, 5) == gm.OK
    assert L.gemm_i4(4, 5, 0, None, 1, None, 3, c, 5) == gm.OK
    assert L.gemm_i4_host(4, 5, 7, a, 3, b, 3, c, 5) == gm.EINVAL  # the host entry point checks the same
    # packing B: ldb counts bytes too
    out = ctypes.c_void_p(0)
    assert L.gemmi_pack_b_i4(7, 5, b, 2, None, ctypes.byref(out)) == gm.EINVAL   # ldb < ceil(5/2)
    assert L.gemmi_pack_b_i4(0, 5, b, 3, None, ctypes.byref(out)) == gm.EINVAL
    assert L.gemmi_pack_b_i4(7, 5, None, 3, None, ctypes.byref(out)) == gm.EINVAL
    assert out.value is None
    # the packed entry point checks its handle and A before any device work
    assert L.gemm_i4_packed(4, a, 4, None, c, 5, None) == gm.EINVAL
    assert L.gemm_i4_packed(-1, a, 4, None, c, 5, None) == gm.EINVAL


def test_options(L):
    old = gm.get_option(gm.OPT_SKINNY_MAX_M)
    gm.set_option(gm.OPT_SKINNY_MAX_M, 4)
    assert gm.get_option(gm.OPT_SKINNY_MAX_M) == 4
    gm.set_option(gm.OPT_SKINNY_MAX_M, old)
    with pytest.raises(gm.GemmiError):
        gm.set_option(gm.OPT_SKINNY_MAX_M, 17)
    with pytest.raises(gm.GemmiError):
        gm.set_option(99, 1)


def test_srs_argument_checks(L):
    dummy = ctypes.c_void_p(0x1000)
    # shift outside [0, 62] is rejected before any device work
    for shift in (-1, 63):
        assert L.gemm_i16_srs(4, 4, 4, dummy, 4, ctypes.c_void_p(0x2000), 4, ctypes.c_void_p(0x3000), 4,
                              shift) == gm.EINVAL
        assert "shift" in gm.last_error()
    assert L.gemm_i16_srs(-1, 4, 4, dummy, 4, dummy, 4, dummy, 4, 0) == gm.EINVAL
    # empty problems are no-ops
    assert L.gemm_i16_srs(0, 4, 4, None, 4, None, 4, None, 4, 3) == gm.OK
    assert L.gemm_i16_srs(3, 3, 0, None, 1, None, 3, ctypes.c_void_p(0x3000), 3, 3) == gm.OK


def test_fused_option(L):
    old = gm.get_option(gm.OPT_FUSED_MAX_N)
    assert old == 64
    gm.set_option(gm.OPT_FUSED_MAX_N, 0)
    assert gm.get_option(gm.OPT_FUSED_MAX_N) == 0
    gm.set_option(gm.OPT_FUSED_MAX_N, old)
    for bad in (-1, 4097):
        with pytest.raises(gm.GemmiError):
            gm.set_option(gm.OPT_FUSED_MAX_N, bad)


def test_pair_option(L):
    assert gm.get_option(gm.OPT_TC_PAIR) == 1
    gm.set_option(gm.OPT_TC_PAIR, 0)
    assert gm.get_option(gm.OPT_TC_PAIR) == 0
    gm.set_option(gm.OPT_TC_PAIR, 1)
    for bad in (-1, 2):
        with pytest.raises(gm.GemmiError):
            gm.set_option(gm.OPT_TC_PAIR, bad)


def test_split_ahead_option(L):
    assert gm.get_option(gm.OPT_SPLIT_AHEAD) == 1
    gm.set_option(gm.OPT_SPLIT_AHEAD, 0)
    assert gm.get_option(gm.OPT_SPLIT_AHEAD) == 0
    gm.set_option(gm.OPT_SPLIT_AHEAD, 1)
    for bad in (-1, 2):
        with pytest.raises(gm.GemmiError):
            gm.set_option(gm.OPT_SPLIT_AHEAD, bad)


def test_conv_rows_option(L):
    assert gm.get_option(gm.OPT_CONV_ROWS) == 1
    gm.set_option(gm.OPT_CONV_ROWS, 0)
    assert gm.get_option(gm.OPT_CONV_ROWS) == 0
    gm.set_option(gm.OPT_CONV_ROWS, 1)
    for bad in (-1, 2):
        with pytest.raises(gm.GemmiError):
            gm.set_option(gm.OPT_CONV_ROWS, bad)


def test_small_problem_option(L):
    assert gm.get_option(gm.OPT_SMALL_MAX_MACS) == 1 << 28
    gm.set_option(gm.OPT_SMALL_MAX_MACS, 0)
    assert gm.get_option(gm.OPT_SMALL_MAX_MACS) == 0
    gm.set_option(gm.OPT_SMALL_MAX_MACS, 1 << 28)
    for bad in (-1, (1 << 40) + 1):
        with pytest.raises(gm.GemmiError):
            gm.set_option(gm.OPT_SMALL_MAX_MACS, bad)


def test_header_constants_match_binding():
    text = open(HEADER).read()
    consts = dict((name, int(v)) for name, v in re.findall(r"GEMMI_((?:OPT|KERNEL)_[A-Z0-9_]+)\s*=\s*(\d+)", text))
    assert consts, "no option or kernel constants found in the header"
    for name, value in consts.items():
        if name == "KERNEL_COUNT":
            assert value == len(gm.KERNELS)
            continue
        assert getattr(gm, name) == value, name
    assert sorted(kid for _, kid in gm.KERNELS) == list(range(consts["KERNEL_COUNT"]))


def test_missing_library_fails_loudly(tmp_path, monkeypatch):
    monkeypatch.setattr(gm, "LIB_PATH", str(tmp_path / "absent.so"))
    monkeypatch.setattr(gm, "_lib", None)
    with pytest.raises(RuntimeError, match="not found"):
        gm.lib()
