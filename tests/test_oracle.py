"""The CPU oracle against what the paper and the mathematics fix (no GPU)."""
import os
import re
import subprocess
import tempfile

import numpy as np
import pytest

import gemm_inputs as gi
import oracle
import oracle_pins as pins


@pytest.fixture(scope="module")
def lib():
    return oracle.load()


def test_golden_hand_cases(lib):
    assert pins.check_golden(lib) == []


@pytest.mark.parametrize("kind", ["i16", "i8"])
def test_bruteforce_tiny_shapes(lib, kind):
    assert pins.check_bruteforce(lib, kinds=(kind,)) == []


def test_extreme_values(lib):
    assert pins.check_extreme_bruteforce(lib) == []


def test_numpy_integer_matmul(lib):
    assert pins.check_numpy(lib) == []


def test_srs_golden(lib):
    assert pins.check_srs_golden(lib) == []


def test_srs_reduces_to_gemm(lib):
    assert pins.check_srs_reduces_to_gemm(lib) == []


def test_srs_closed_forms(lib):
    assert pins.check_srs_closed_forms(lib) == []


def test_srs_rejects_bad_shift(lib):
    A = np.ones((2, 3), np.int16)
    B = np.ones((3, 2), np.int16)
    for shift in (-1, 63):
        with pytest.raises(ValueError):
            oracle.gemm_srs(A, B, np.zeros((2, 2), np.int16), shift, lib=lib)


def test_conv_golden(lib):
    assert pins.check_conv_golden(lib) == []


def test_conv_1x1_is_gemm(lib):
    assert pins.check_conv_1x1_is_gemm(lib) == []


def test_conv_delta_kernels(lib):
    assert pins.check_conv_delta_kernels(lib) == []


def test_conv_im2col_lowering(lib):
    assert pins.check_conv_im2col_lowering(lib) == []


def test_i4_golden(lib):
    assert pins.check_i4_golden(lib) == []


def test_i4_bruteforce_tiny_shapes(lib):
    assert pins.check_i4_bruteforce(lib) == []


def test_i4_matches_i8_and_numpy(lib):
    assert pins.check_i4_matches_i8(lib) == []


def test_i4_closed_forms(lib):
    assert pins.check_i4_closed_forms(lib) == []


def test_i4_packer_matches_golden_bytes():
    """The shared packer stores the format the hand-worked cases spell out byte by byte."""
    v = np.array([[1, 2, -1, -8, 3]], np.int8)
    assert gi.pack_nibbles(v).tolist() == [[0x21, 0x8F, 0x03]]
    assert gi.pack_nibbles(v, ld=4, pad=0x55).tolist() == [[0x21, 0x8F, 0x53, 0x55]]


def test_i4_packer_rejects_bad_input():
    with pytest.raises(ValueError):
        gi.pack_nibbles(np.array([[8]], np.int8))           # outside [-8, 7]
    with pytest.raises(ValueError):
        gi.pack_nibbles(np.array([[-9, 0]], np.int8))
    with pytest.raises(ValueError):
        gi.pack_nibbles(np.zeros((2, 5), np.int8), ld=2)    # pitch below ceil(5/2) = 3 bytes
    assert gi.pack_nibbles(np.zeros((0, 5), np.int8)).shape == (0, 3)


def test_i4_invalid_arguments_rejected(lib):
    b = np.zeros((4, 4), np.uint8)
    c = np.zeros((4, 4), np.int32)
    f = lib.gemm_oracle_i4
    p, q = b.ctypes.data, c.ctypes.data
    assert f(2, 3, 3, p, 2, p, 2, q, 3, 1) == 0
    assert f(2, 3, 3, p, 1, p, 2, q, 3, 1) == 1   # lda < ceil(k/2)
    assert f(2, 3, 3, p, 2, p, 1, q, 3, 1) == 1   # ldb < ceil(n/2)
    assert f(2, 3, 3, p, 2, p, 2, q, 2, 1) == 1   # ldc < n
    assert f(2, 3, 3, 0, 2, p, 2, q, 3, 1) == 1   # null A
    assert f(2, 3, 0, 0, 0, 0, 0, q, 3, 1) == 0   # k = 0: C unchanged, A and B unused


def test_closed_forms(lib):
    assert pins.check_closed_forms(lib) == []


def test_identity_and_permutation(lib):
    assert pins.check_identity_permutation(lib) == []


def test_blocked_algorithm_equivalence(lib):
    assert pins.check_blocked(lib) == []


def test_padding_untouched(lib):
    assert pins.check_padding(lib) == []


def test_linearity(lib):
    assert pins.check_linearity(lib) == []


def test_transpose_identity(lib):
    assert pins.check_transpose(lib) == []


def test_zero_sizes_and_k0(lib):
    A, B, C = gi.random_problem(5, 4, 6, 0, "i16")
    X = C.copy()
    oracle.gemm(A, B, X, lib=lib)
    assert np.array_equal(X, C)
    for m, n in ((0, 5), (5, 0), (0, 0)):
        A, B, C = gi.random_problem(6, m, n, 3, "i16")
        oracle.gemm(A, B, C, lib=lib)


def test_invalid_arguments_rejected(lib):
    i64 = np.zeros((2, 2), np.int64)
    a = np.zeros((2, 2), np.int16)
    f = lib.gemm_oracle_i16
    p = a.ctypes.data
    c = i64.ctypes.data
    assert f(-1, 2, 2, p, 2, p, 2, c, 2, 1) == 1
    assert f(2, 2, 2, p, 1, p, 2, c, 2, 1) == 1   # lda < k
    assert f(2, 2, 2, p, 2, p, 1, c, 2, 1) == 1   # ldb < n
    assert f(2, 2, 2, p, 2, p, 2, c, 1, 1) == 1   # ldc < n
    assert f(2, 2, 2, 0, 2, p, 2, c, 2, 1) == 1   # null A
    assert f(2, 2, 2, p, 2, p, 2, c, 2, 1) == 0


def test_threads_do_not_change_result(lib):
    A, B, C = gi.random_problem(12, 97, 33, 65, "i16")
    X1, X4 = C.copy(), C.copy()
    oracle.gemm(A, B, X1, nthreads=1, lib=lib)
    oracle.gemm(A, B, X4, nthreads=4, lib=lib)
    assert np.array_equal(X1, X4)


def test_workload_small_case_matches_numpy(lib):
    """The 256^3 workload (C in [-2^20, 2^20]) against numpy's exact int64 matmul."""
    w = gi.WORKLOADS["i16_256"]
    A, B, C = gi.make_inputs(w)
    X = C.copy()
    oracle.gemm(A, B, X, nthreads=4, lib=lib)
    assert np.array_equal(X, pins.numpy_gemm(A, B, C))


# --- mutation tests: a mistake planted in a copy of the oracle must be caught ---

MUTANTS = {
    "drop_last_rank1_term": ("for (int64_t p = 0; p < k; ++p) {", "for (int64_t p = 0; p < k - 1; ++p) {"),
    "wrong_sign": ("c[j] += (uint64_t)(a * (int64_t)b[j]);", "c[j] -= (uint64_t)(a * (int64_t)b[j]);"),
    # an indexing mistake that stays inside A (a transposed index can read past it and crash)
    "reversed_A_index": ("const int64_t a = (int64_t)A[i * lda + p];", "const int64_t a = (int64_t)A[i * lda + (k - 1 - p)];"),
    "int32_accumulator": ("c[j] += (uint64_t)(a * (int64_t)b[j]);",
                          "c[j] = (uint64_t)(int64_t)(int32_t)(uint32_t)(c[j] + (uint64_t)(a * (int64_t)b[j]));"),
    "overwrites_C": ("uint64_t* c = (uint64_t*)(C + i * ldc);",
                     "uint64_t* c = (uint64_t*)(C + i * ldc); for (int64_t q = 0; q < n; ++q) c[q] = 0;"),
    "ignores_ldb": ("const int16_t* b = B + p * ldb;", "const int16_t* b = B + p * n;"),
    "off_by_one_column": ("for (int64_t j = 0; j < n; ++j)\n        c[j] +=", "for (int64_t j = 1; j < n; ++j)\n        c[j] +="),
    "i8_truncates_to_16_bits": ("c[j] += (uint32_t)(a * (int32_t)b8[j]);",
                                "c[j] = (uint16_t)(c[j] + (uint32_t)(a * (int32_t)b8[j]));"),
    "i8_drops_last_term": ("for (int64_t p = 0; p < k; ++p) {\n      /* one rank-1 term, as in the int16 loop",
                           "for (int64_t p = 0; p + 1 < k; ++p) {\n      /* one rank-1 term, as in the int16 loop"),
    "i8_wrong_sign": ("c[j] += (uint32_t)(a * (int32_t)b8[j]);", "c[j] -= (uint32_t)(a * (int32_t)b8[j]);"),
    "i8_transposed_B": ("c[j] += (uint32_t)(a * (int32_t)b8[j]);", "c[j] += (uint32_t)(a * (int32_t)B[j * ldb + p]);"),
    # the micro-kernel output C16 += srs(A*B, shift)
    "srs_rounds_half_down": ("oracle_floor_div_pow2(s + ((int64_t)1 << (shift - 1)), shift)",
                             "oracle_floor_div_pow2(s + ((int64_t)1 << (shift - 1)) - 1, shift)"),
    "srs_truncates_toward_zero": ("  if (v >= 0) return v / d;\n  return -((-v + d - 1) / d);", "  return v / d;"),
    "srs_no_positive_saturation": ("if (r > 32767) r = 32767;", "if (r > 65535) r = 65535;"),
    "srs_no_negative_saturation": ("if (r < -32768) r = -32768;", "if (r < -65536) r = -65536;"),
    "srs_saturating_add": ("const uint16_t sum = (uint16_t)((uint16_t)C[i * ldc + j] + (uint16_t)r);",
                           "int64_t t = (int64_t)C[i * ldc + j] + r; if (t > 32767) t = 32767; "
                           "if (t < -32768) t = -32768; const uint16_t sum = (uint16_t)t;"),
    "srs_overwrites_C": ("(uint16_t)((uint16_t)C[i * ldc + j] + (uint16_t)r)", "(uint16_t)r"),
    "srs_shift_off_by_one": ("const int64_t d = (int64_t)1 << shift;", "const int64_t d = (int64_t)1 << (shift + 1);"),
    "srs_drops_last_term": ("for (int64_t p = 0; p < k; ++p) s +=", "for (int64_t p = 0; p + 1 < k; ++p) s +="),
    # the convolution through the lowered GEMM
    "conv_swaps_r_and_s": ("const int16_t* wt = Wt + ((r * S + s) * Cin + c) * Cout;",
                           "const int16_t* wt = Wt + ((s * R + r) * Cin + c) * Cout;"),
    "conv_padding_off_by_one": ("const int64_t h = ho + r - pad_h;", "const int64_t h = ho + r - pad_h + 1;"),
    "conv_wraps_instead_of_zero_padding": ("const int64_t w = wo + s - pad_w;",
                                           "const int64_t w = (wo + s - pad_w + W) % W;"),
    "conv_drops_last_channel": ("for (int64_t c = 0; c < Cin; ++c) {\n            const int64_t a = (int64_t)x[c];",
                                "for (int64_t c = 0; c + 1 < Cin; ++c) {\n            const int64_t a = (int64_t)x[c];"),
    # the int4 variant
    "i4_nibble_order_swapped": ("(idx % 2 == 0) ? (byte & 15u) : (byte >> 4)", "(idx % 2 == 0) ? (byte >> 4) : (byte & 15u)"),
    "i4_unsigned_nibbles": ("return v >= 8 ? (int64_t)v - 16 : (int64_t)v;", "return (int64_t)v;"),
    "i4_sign_threshold_off_by_one": ("return v >= 8 ? (int64_t)v - 16 : (int64_t)v;", "return v > 8 ? (int64_t)v - 16 : (int64_t)v;"),
    "i4_row_pitch_in_elements": ("oracle_nibble(A + i * lda, p)", "oracle_nibble(A + i * lda / 2, p)"),
    "i4_ignores_ldb": ("oracle_nibble(B + p * ldb, j)", "oracle_nibble(B + p * ((n + 1) / 2), j)"),
    "i4_drops_last_term": ("for (int64_t p = 0; p < k; ++p)\n        s += (uint64_t)(oracle_nibble",
                           "for (int64_t p = 0; p + 1 < k; ++p)\n        s += (uint64_t)(oracle_nibble"),
    "i4_wraps_at_16_bits": ("s += (uint64_t)(oracle_nibble(A + i * lda, p) * oracle_nibble(B + p * ldb, j));\n      c[j] = (int32_t)(uint32_t)s;",
                            "s += (uint64_t)(oracle_nibble(A + i * lda, p) * oracle_nibble(B + p * ldb, j));\n      c[j] = (int32_t)(int16_t)s;"),
    "conv_channel_stride_is_cout": ("const int16_t* x = X + ((n * H + h) * W + w) * Cin;",
                                    "const int16_t* x = X + ((n * H + h) * W + w) * Cout;"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_planted_mistake_is_caught(name):
    src = open(os.path.join(os.path.dirname(oracle.__file__), "gemm_oracle.c")).read()
    old, new = MUTANTS[name]
    assert src.count(old) >= 1, f"mutation anchor not found: {old!r}"
    mutated = src.replace(old, new, 1)
    with tempfile.TemporaryDirectory() as d:
        s = os.path.join(d, "mut.c")
        so = os.path.join(d, "libmut.so")
        open(s, "w").write(mutated)
        subprocess.run(["gcc", "-O1", "-std=c11", "-shared", "-fPIC", s, "-o", so], check=True,
                       capture_output=True)
        lib = oracle.load(so)
        small = [(m, n, k) for m in (1, 2, 5) for n in (1, 3, 8) for k in (1, 2, 17)]
        failures = pins.pin_failures(lib, bruteforce_shapes=small)
    assert failures, f"mutant {name} passed every pin"
