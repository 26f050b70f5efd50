"""GPU parity of gemmi_conv2d_i16: a convolution through the lowered GEMM (IM2COL).

"Same" stride-1 convolutions with 64 input channels (odd R and S, one exact chunk,
an even Cout, padded rows of at most 128 pixels) run the direct kernel
(conv_rows.cu), which splits every input pixel once; other "same" convolutions
with Cin % 64 == 0 run the fused kernel directly on the NHWC tensor (the lowered
matrix is never formed); other shapes lower X with im2col.cu first.  Expected
values come from the oracle's direct convolution (oracle.conv2d) on the same
seeded inputs, bit for bit.
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


def direct_applies(gm, shape):
    """Whether gemmi_conv2d_i16 takes the direct kernel for this shape (aligned tensors, default
    options otherwise): the rule of the library's dispatch, restated."""
    N, H, W, Ci, Co, R, S, ph, pw = shape
    if gm.get_option(gm.OPT_CONV_ROWS) == 0 or Ci != 64 or R % 2 == 0 or S % 2 == 0:
        return False
    if 2 * ph != R - 1 or 2 * pw != S - 1 or Co % 2 or Co > 64 or N * H * W <= gm.get_option(gm.OPT_SKINNY_MAX_M):
        return False
    if R * S > 12 or R * S * 64 > 512 * gm.get_option(gm.OPT_TC_CHUNK_SCALE):
        return False
    wp, wpad = W + S - 1, (W + 7) // 8 * 8
    if wp > 128 or min(128 // wp, 120 // wpad) < 1:
        return False
    return (128 + (R - 1) * wp + (S - 1) + 7) // 8 * 8 <= 256


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


@pytest.fixture
def conv_rows_option(gm, request):
    gm.set_option(gm.OPT_CONV_ROWS, request.param)
    yield request.param
    gm.set_option(gm.OPT_CONV_ROWS, 1)


@pytest.mark.parametrize("conv_rows_option", [1, 0], indirect=True, ids=["direct_on", "direct_off"])
@pytest.mark.parametrize("shape", IMPLICIT)
def test_conv_implicit(gm, shape, conv_rows_option):
    N, H, W, Ci, Co, R, S, ph, pw = shape
    X, Wt, Y = make(900 + sum(shape), *shape)
    got, counts = run(gm, X, Wt, Y, R, S, ph, pw)
    kernel = "conv_rows" if direct_applies(gm, shape) else "fused_i16"
    assert counts[kernel] == 1, (kernel, counts)
    assert counts["tc_i16"] + counts["tc_pair_i16"] + counts["tc_pair_i16_ahead"] == 0, counts
    assert counts["conv_rows"] + counts["fused_i16"] == 1, counts
    assert_same(got, expected(X, Wt, Y, R, S, ph, pw), f"implicit {shape}")


# shapes at the edges of the direct kernel's rule, and a few just beyond it (the fused kernel)
DIRECT_EDGES = [
    (1, 5, 61, 64, 64, 3, 3, 1, 1),     # padded row of 63: the largest 3x3 window buffer (256 positions)
    (1, 5, 62, 64, 64, 3, 3, 1, 1),     # padded row of 64: beyond the buffer -> fused kernel
    (2, 6, 7, 64, 2, 3, 3, 1, 1),       # two output channels
    (2, 5, 9, 64, 130, 3, 3, 1, 1),     # more than 64 output channels -> fused kernel
    (1, 4, 12, 64, 256, 3, 3, 1, 1),    # four channel blocks -> fused kernel
    (3, 5, 8, 64, 48, 5, 3, 2, 1),      # 5x3: 15 taps -> fused kernel
    (2, 6, 20, 64, 40, 1, 5, 0, 2),     # 1x5, 40 output channels
    (2, 7, 9, 64, 34, 3, 3, 1, 1),      # 34 output channels: a partial group of 16
    (2, 7, 20, 64, 64, 1, 3, 0, 1),     # 1x3
    (1, 3, 120, 64, 64, 1, 3, 0, 1),    # one output row of 120 pixels per tile (the staging limit)
    (1, 3, 121, 64, 64, 1, 3, 0, 1),    # 121 pixels: beyond the staging limit -> fused kernel
    (2, 6, 8, 64, 63, 3, 3, 1, 1),      # odd Cout -> fused kernel
    (5, 20, 3, 64, 64, 3, 3, 1, 1),     # narrow images, 17 rows per tile, ragged last tile
]


@pytest.mark.parametrize("shape", DIRECT_EDGES)
def test_conv_direct_edges(gm, shape):
    N, H, W, Ci, Co, R, S, ph, pw = shape
    X, Wt, Y = make(1100 + sum(shape), *shape)
    got, counts = run(gm, X, Wt, Y, R, S, ph, pw)
    kernel = "conv_rows" if direct_applies(gm, shape) else "fused_i16"
    assert counts[kernel] == 1, (kernel, counts)
    assert_same(got, expected(X, Wt, Y, R, S, ph, pw), f"direct edge {shape}")


def test_conv_direct_chunk_scale_one(gm):
    """At chunk scale 1 a 3x3 filter (576 reduction indices) exceeds one exact chunk, so the fused
    kernel takes it; a 1x1 filter still runs direct.  Both exact."""
    gm.set_option(gm.OPT_TC_CHUNK_SCALE, 1)
    try:
        for shape, kernel in (((2, 6, 9, 64, 64, 3, 3, 1, 1), "fused_i16"), ((2, 6, 9, 64, 64, 1, 1, 0, 0), "conv_rows")):
            N, H, W, Ci, Co, R, S, ph, pw = shape
            X, Wt, Y = make(1200 + sum(shape), *shape)
            got, counts = run(gm, X, Wt, Y, R, S, ph, pw)
            assert counts[kernel] == 1, (shape, counts)
            assert_same(got, expected(X, Wt, Y, R, S, ph, pw), f"chunk scale 1 {shape}")
    finally:
        gm.set_option(gm.OPT_TC_CHUNK_SCALE, 2)


def test_conv_direct_every_int16_value(gm):
    """Every int16 value passes through the direct kernel's on-chip split: X holds all 65536
    values (64 channels x 1024 pixels), against weights with extreme and ragged values."""
    X = np.arange(-32768, 32768, dtype=np.int64).astype(np.int16).reshape(1, 16, 64, 64)
    Wt = gi.uniform_int(1301, (9 * 64, 64), -32768, 32767, np.int16)
    Wt[0, :] = -32768
    Wt[1, :] = 32767
    Y = np.zeros((1, 16, 64, 64), np.int64)
    # W = 64 needs a padded row of 66 > 63: run it as 1x3 (padded row 66, window 128 + 2)
    Wt13 = Wt[:3 * 64].copy()
    got, counts = run(gm, X, Wt13, Y, 1, 3, 0, 1)
    assert counts["conv_rows"] == 1, counts
    assert_same(got, expected(X, Wt13, Y, 1, 3, 0, 1), "every int16 value, 1x3")
    X2 = X.reshape(1, 32, 32, 64)
    Y2 = np.zeros((1, 32, 32, 64), np.int64)
    got, counts = run(gm, X2, Wt, Y2, 3, 3, 1, 1)
    assert counts["conv_rows"] == 1, counts
    assert_same(got, expected(X2, Wt, Y2, 3, 3, 1, 1), "every int16 value, 3x3")


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


@pytest.mark.parametrize("conv_rows_option", [1, 0], indirect=True, ids=["direct", "fused"])
def test_conv_workload_every_element(gm, conv_rows_option):
    """The convolution of the im2col workload (batch 32, 56x56, 64 -> 64 channels, 3x3, pad 1),
    run whole on the direct kernel and on the fused one; every element against the oracle."""
    N, H, W, Ci, Co = 32, 56, 56, 64, 64
    X, Wt, _ = make(1003, N, H, W, Ci, Co, 3, 3, 1, 1, dist="conv")
    Y = gi.uniform_int(1004, (N, H, W, Co), -(1 << 40), 1 << 40, np.int64)
    got, counts = run(gm, X, Wt, Y, 3, 3, 1, 1)
    assert counts["conv_rows" if conv_rows_option else "fused_i16"] == 1, counts
    Z = Y.copy()
    oracle.conv2d(X, Wt, Z, 3, 3, 1, 1, nthreads=oracle.host_cores())
    assert_same(got, Z, "conv workload")


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


def _random_conv_shapes(count, seed):
    """Seeded random convolution shapes over the three paths: "same" 64-channel convolutions with
    odd filters (the direct kernel when its rule holds), other "same" ones with Cin % 64 == 0 (the
    fused kernel on the NHWC tensor) and everything else (lowered first).  The oracle's work per
    case stays below about 4e7 multiply-adds."""
    rng = np.random.Generator(np.random.Philox(seed))
    shapes = []
    while len(shapes) < count:
        kind = len(shapes) % 3
        R = int(rng.choice([1, 3, 5])) if kind < 2 else int(rng.integers(1, 5))
        S = int(rng.choice([1, 3, 5])) if kind < 2 else int(rng.integers(1, 5))
        if kind == 0:
            Ci, ph, pw = 64, (R - 1) // 2, (S - 1) // 2
            Co = int(rng.integers(1, 33)) * 2
        elif kind == 1:
            Ci, ph, pw = int(rng.choice([64, 128])), (R - 1) // 2, (S - 1) // 2
            Co = int(rng.integers(1, 80))
        else:
            Ci = int(rng.choice([3, 8, 16, 40, 64]))
            ph, pw = int(rng.integers(0, R)), int(rng.integers(0, S))
            Co = int(rng.integers(1, 70))
        N = int(rng.integers(1, 4))
        H = int(rng.integers(1, 30))
        W = int(rng.choice([int(rng.integers(1, 40)), int(rng.integers(100, 121))]))
        Ho, Wo = H + 2 * ph - R + 1, W + 2 * pw - S + 1
        if Ho < 1 or Wo < 1 or N * Ho * Wo * Co * R * S * Ci > 4e7:
            continue
        shapes.append((N, H, W, Ci, Co, R, S, ph, pw))
    return shapes


RANDOM_CONV = _random_conv_shapes(45, 2302)


@pytest.mark.parametrize("shape", RANDOM_CONV, ids=lambda s: "x".join(map(str, s)))
def test_conv_random_sweep(gm, shape):
    """Every element of a seeded random convolution against the oracle; where the direct kernel's
    rule holds, that kernel is the one that ran."""
    N, H, W, Ci, Co, R, S, ph, pw = shape
    X, Wt, Y = make(9300 + sum(shape) * 7, *shape)
    got, counts = run(gm, X, Wt, Y, R, S, ph, pw)
    if direct_applies(gm, shape):
        assert counts["conv_rows"] == 1, counts
    else:
        assert counts["conv_rows"] == 0, counts
    assert_same(got, expected(X, Wt, Y, R, S, ph, pw), f"random {shape}")
