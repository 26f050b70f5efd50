"""The seeded input generator shared by the oracle and the CUDA path (no GPU)."""
import numpy as np

import gemm_inputs as gi


def test_splitmix64_published_sequence():
    # First outputs of SplitMix64 started at state 0 (Steele, Lea, Flood 2014;
    # the sequence used to seed the xoshiro/xorshift family).
    r = gi.splitmix64(0, 0, 3)
    assert [int(x) for x in r] == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]


def test_counter_based_offsets():
    full = gi.splitmix64(123, 0, 1000)
    assert np.array_equal(gi.splitmix64(123, 400, 100), full[400:500])


def test_ranges_and_types():
    a = gi.uniform_int(5, (1000, 1000), -32768, 32767, np.int16)
    assert a.dtype == np.int16 and a.min() == -32768 and a.max() == 32767
    b = gi.uniform_int(6, (1000,), -2048, 2047, np.int16)
    assert b.min() >= -2048 and b.max() <= 2047
    z = gi.half_zero_uniform(7, (200000,), 4095, np.int16)
    frac0 = float((z == 0).mean())
    assert 0.49 < frac0 < 0.51 and z.min() == 0 and z.max() == 4095


def test_row_slices_match_full_matrix():
    w = gi.WORKLOADS["i16_256"]
    A, B, C = gi.make_inputs(w)
    A2, B2, C2 = gi.make_inputs(w, rows=slice(100, 140))
    assert np.array_equal(A[100:140], A2) and np.array_equal(B, B2) and np.array_equal(C[100:140], C2)
    assert C.min() >= -(1 << 20) and C.max() <= (1 << 20)


def test_workload_table():
    w = gi.WORKLOADS
    assert (w["conv3x3_im2col"].m, w["conv3x3_im2col"].n, w["conv3x3_im2col"].k) == (32 * 56 * 56, 64, 64 * 9)
    assert w["i8_4096"].kind == "i8" and w["i16_8192"].ops == 2 * 8192 ** 3
    assert (w["skinny_8x4096x4096"].m, w["skinny_8x4096x4096"].n) == (8, 4096)
