"""GPU parity of gemmi_conv2d_i16: a convolution through the lowered GEMM (IM2COL).

"Same" stride-1 convolutions with Cin % 64 == 0 run the fused kernel directly on
the NHWC tensor (the lowered matrix is never formed); other shapes lower X with
im2col.cu first.  Expected values come from the oracle's direct convolution
(oracle.conv2d) on the same seeded inputs, bit for bit.
"""
import numpy as np
import pytest

import gemm_inputs as gi
import oracle

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def gm():
    import paper_2302_07594_gb300 as gm
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    gm.lib()
    return gm


def make(seed, N, H, W, Cin, Cout, R, S, ph, pw, dist="full"):
    Ho, Wo = H + 2 * ph - R + 1, W + 2 * pw - S + 1
    if dist == "conv":  # the conv workload's activations: half exact zeros, else [0, 4095]
        X = gi.half_zero_uniform(seed, (N, H, W, Cin), 4095, np.int16)
        Wt = gi.uniform_int(seed + 1, (R * S * Cin, Cout), -2048, 2047, np.int16)
    else:
        X = gi.uniform_int(seed, (N, H, W, Cin), -32768, 32767, np.int16)
        Wt = gi.uniform_int(seed + 1, (R * S * Cin, Cout), -32768, 32767, np.int16)
    Y = gi.uniform_int(seed + 2, (N, Ho, Wo, Cout), -(1 << 40), 1 << 40, np.int64)
    return X, Wt, Y


def run(gm, X, Wt, Y, R, S, ph, pw):
    dX, dW, dY = (torch.from_numpy(np.ascontiguousarray(t)).cuda() for t in (X, Wt, Y))
    gm.kernel_timing(True)
    try:
        gm.conv2d_i16(dX, dW, dY, R, S, ph, pw)
        torch.cuda.synchronize()
        counts = {name: gm.kernel_time(kid)[1] for name, kid in gm.KERNELS}
    finally:
        gm.kernel_timing(False)
    assert gm.device_status() == gm.OK
    return dY.cpu().numpy(), counts


def expected(X, Wt, Y, R, S, ph, pw):
    Z = Y.copy()
    oracle.conv2d(X, Wt, Z, R, S, ph, pw, nthreads=8)
    return Z


def assert_same(got, exp, what=""):
    if not np.array_equal(got, exp):
        bad = np.argwhere(got != exp)
        raise AssertionError(f"{what}: {len(bad)} mismatches, first at {tuple(bad[0])}: "
                             f"got {got[tuple(bad[0])]} want {exp[tuple(bad[0])]}")


# (N, H, W, Cin, Cout, R, S, pad_h, pad_w): "same" convolutions with Cin % 64 == 0 -> implicit path
IMPLICIT = [
    (2, 9, 11, 64, 64, 3, 3, 1, 1),     # ragged last tile, taps crossing image rows and images
    (1, 56, 56, 64, 64, 3, 3, 1, 1),    # one image of the conv workload
    (3, 7, 5, 128, 40, 3, 3, 1, 1),     # two channel blocks per tap, a partial output tile
    (1, 12, 13, 64, 100, 5, 5, 2, 2),   # 5x5, two output tiles
    (2, 10, 10, 64, 64, 1, 1, 0, 0),    # 1x1
    (2, 9, 6, 64, 32, 3, 1, 1, 0),      # 3x1
    (4, 1, 40, 64, 64, 3, 3, 1, 1),     # one-row images: every vertical tap but the middle is padding
    (3, 40, 1, 64, 64, 3, 3, 1, 1),     # one-column images
]


@pytest.mark.parametrize("shape", IMPLICIT)
def test_conv_implicit(gm, shape):
    N, H, W, Ci, Co, R, S, ph, pw = shape
    X, Wt, Y = make(900 + sum(shape), *shape)
    got, counts = run(gm, X, Wt, Y, R, S, ph, pw)
    assert counts["fused_i16"] == 1 and counts["tc_i16"] + counts["tc_pair_i16"] + counts["tc_pair_i16_ahead"] == 0, counts
    assert_same(got, expected(X, Wt, Y, R, S, ph, pw), f"implicit {shape}")


FALLBACK = [
    (2, 9, 11, 3, 16, 3, 3, 1, 1),      # Cin not a multiple of 64
    (1, 10, 12, 64, 64, 3, 3, 0, 0),    # valid convolution: output smaller than the input
    (2, 6, 7, 8, 300, 3, 3, 1, 1),      # wide output: general tensor-core path
    (1, 3, 4, 5, 7, 2, 3, 1, 0),        # tiny: skinny path (output rows <= 16)
]


@pytest.mark.parametrize("shape", FALLBACK)
def test_conv_lowered_fallback(gm, shape):
    N, H, W, Ci, Co, R, S, ph, pw = shape
    X, Wt, Y = make(950 + sum(shape), *shape)
    got, counts = run(gm, X, Wt, Y, R, S, ph, pw)
    assert_same(got, expected(X, Wt, Y, R, S, ph, pw), f"fallback {shape}")


def test_conv_extremes(gm):
    for a, b in ((-32768, -32768), (32767, -32768), (32767, 32767)):
        X = np.full((2, 8, 9, 64), a, np.int16)
        Wt = np.full((9 * 64, 64), b, np.int16)
        Y = np.zeros((2, 8, 9, 64), np.int64)
        got, _ = run(gm, X, Wt, Y, 3, 3, 1, 1)
        assert_same(got, expected(X, Wt, Y, 3, 3, 1, 1), f"constant {(a, b)}")


def test_conv_workload_images(gm):
    """The convolution of the im2col workload (batch 32, 56x56, 64 -> 64 channels, 3x3, pad 1),
    run whole; the oracle checks images 0, 13 and 31 (images are independent)."""
    N, H, W, Ci, Co = 32, 56, 56, 64, 64
    X, Wt, _ = make(1003, N, H, W, Ci, Co, 3, 3, 1, 1, dist="conv")
    Y = np.zeros((N, H, W, Co), np.int64)
    got, counts = run(gm, X, Wt, Y, 3, 3, 1, 1)
    assert counts["fused_i16"] == 1, counts
    for n in (0, 13, 31):
        exp = expected(X[n:n + 1].copy(), Wt, Y[n:n + 1].copy(), 3, 3, 1, 1)
        assert_same(got[n:n + 1], exp, f"image {n}")


def test_conv_argument_errors(gm):
    dX = torch.zeros((1, 4, 4, 64), dtype=torch.int16, device="cuda")
    dW = torch.zeros((9 * 64, 8), dtype=torch.int16, device="cuda")
    dY = torch.zeros((1, 4, 4, 8), dtype=torch.int64, device="cuda")
    with pytest.raises(ValueError):
        gm.conv2d_i16(dX, dW, dY, 3, 3, 0, 0)  # Y has the wrong shape for a valid convolution
    L = gm.lib()
    assert L.gemmi_conv2d_i16(1, 4, 4, 64, 8, 0, 3, 1, 1, dX.data_ptr(), dW.data_ptr(), dY.data_ptr(), None) == gm.EINVAL
    assert L.gemmi_conv2d_i16(1, 2, 2, 64, 8, 5, 5, 0, 0, dX.data_ptr(), dW.data_ptr(), dY.data_ptr(), None) == gm.EINVAL
    # an empty output is a no-op
    assert L.gemmi_conv2d_i16(0, 4, 4, 64, 8, 3, 3, 1, 1, None, None, None, None) == gm.OK
