"""GPU parity of the overlapped A split (GEMMI_OPT_SPLIT_AHEAD) against the oracle, bit for bit.

With the option on (the default), an int16 GEMM on SM pairs splits B and only the row panels of A
that the first wave of tiles reads before the GEMM kernel; two warps of every CTA of the pair
kernel split the remaining panels (128 rows x 256 reduction indices per work item) while the
tensor cores work, and each tile's loads wait until its panel is complete.  These tests cover:
ragged last panels (m % 128 != 0) and ragged last reduction items (k % 256 != 0), a narrow output
(n of two tile columns) whose first wave spans several raster bands, every int16 value of A
through the splitter warps, both exact-chunk lengths, weights packed once, calls of different
sizes in a row (the work counters start from zero every call), the option switched off, and the
layouts that keep the whole split in front (k % 8 != 0).  Which kernel ran is read back from the
library's per-kernel launch counters.
"""
import numpy as np
import pytest

import gemm_inputs as gi
import oracle

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

# (m, n, k): every one has more row panels than the first wave of tiles reads
AHEAD_SHAPES = [(2100, 1280, 1000), (6000, 136, 264), (4096, 2048, 512), (2048, 1408, 8)]


@pytest.fixture(scope="module")
def gm():
    import paper_2302_07594_gb300 as gm
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    gm.lib()
    assert gm.get_option(gm.OPT_SPLIT_AHEAD) == 1
    assert gm.get_option(gm.OPT_TC_PAIR) == 1
    yield gm
    gm.set_option(gm.OPT_SPLIT_AHEAD, 1)


@pytest.fixture(params=[1, 2], ids=["chunks_2^23", "chunks_2^24"])
def chunk_scale(request, gm):
    old = gm.get_option(gm.OPT_TC_CHUNK_SCALE)
    gm.set_option(gm.OPT_TC_CHUNK_SCALE, request.param)
    yield request.param
    gm.set_option(gm.OPT_TC_CHUNK_SCALE, old)


def expected(A, B, C):
    X = C.copy()
    oracle.gemm(A, B, X, nthreads=oracle.host_cores())
    return X


def counts_of(gm, fn):
    gm.kernel_timing(True)
    try:
        fn()
        torch.cuda.synchronize()
        return {name: gm.kernel_time(kid)[1] for name, kid in gm.KERNELS}
    finally:
        gm.kernel_timing(False)


def run(gm, A, B, C, expect_ahead=True):
    dA, dB, dC = (torch.from_numpy(np.ascontiguousarray(x)).cuda() for x in (A, B, C))
    counts = counts_of(gm, lambda: gm.gemm_i16(dA, dB, dC))
    assert gm.device_status() == gm.OK
    assert counts["tc_pair_i16_ahead"] == (1 if expect_ahead else 0), counts
    assert counts["tc_pair_i16"] == (0 if expect_ahead else 1), counts
    assert counts["split"] == 1, counts
    return dC.cpu().numpy()


def assert_same(got, exp, what):
    if not np.array_equal(got, exp):
        bad = np.argwhere(got != exp)
        r, c = bad[0]
        raise AssertionError(f"{what}: {len(bad)} elements differ, first at ({r}, {c}): "
                             f"got {got[r, c]}, expected {exp[r, c]}")


@pytest.mark.parametrize("shape", AHEAD_SHAPES, ids=lambda s: "x".join(map(str, s)))
def test_ahead_every_element(gm, chunk_scale, shape):
    m, n, k = shape
    A, B, C = gi.random_problem(7100 + m + k, m, n, k, "i16")
    assert_same(run(gm, A, B, C), expected(A, B, C), f"{shape} chunk scale {chunk_scale}")


def test_ahead_every_int16_value_of_A(gm):
    """All 65536 int16 values appear in A (16 times each, shuffled) and go through the splitter
    warps' byte logic: every row panel past the first wave is split inside the GEMM kernel."""
    m, n, k = 4096, 1280, 256
    vals = np.arange(-32768, 32768, dtype=np.int64)
    A = np.tile(vals, m * k // vals.size)
    rng = np.random.Generator(np.random.Philox(91))
    A = A[rng.permutation(A.size)].astype(np.int16).reshape(m, k)
    _, B, C = gi.random_problem(7201, m, n, k, "i16")
    assert_same(run(gm, A, B, C), expected(A, B, C), "every int16 value")


def test_ahead_extreme_constants(gm, chunk_scale):
    m, n, k = 2176, 1280, 1024
    for a, b in ((-32768, -32768), (32767, -32768), (-32768, 32767), (32767, 32767)):
        A = np.full((m, k), a, np.int16)
        B = np.full((k, n), b, np.int16)
        C = np.zeros((m, n), np.int64)
        exp = np.full((m, n), a * b * k, np.int64)
        assert_same(run(gm, A, B, C), exp, f"constant {a} x {b}")


def test_ahead_calls_of_different_sizes_in_a_row(gm):
    """The claim and completion counters are zeroed by every call: a smaller call after a larger
    one (fewer panels, other items per panel) and the larger one again."""
    for i, shape in enumerate([(6000, 1280, 1000), (2100, 1408, 264), (6000, 1280, 1000)]):
        m, n, k = shape
        A, B, C = gi.random_problem(7300 + i, m, n, k, "i16")
        assert_same(run(gm, A, B, C), expected(A, B, C), f"call {i} {shape}")


def test_ahead_packed_weights(gm):
    m, n, k = 2100, 1280, 1000
    A, B, C = gi.random_problem(7400, m, n, k, "i16")
    Bp = gm.pack_b_i16(torch.from_numpy(B).cuda())
    dA, dC = torch.from_numpy(A).cuda(), torch.from_numpy(C).cuda()
    counts = counts_of(gm, lambda: gm.gemm_i16_packed(dA, Bp, dC))
    assert gm.device_status() == gm.OK
    assert counts["tc_pair_i16_ahead"] == 1 and counts["tc_pair_i16"] == 0, counts
    assert_same(dC.cpu().numpy(), expected(A, B, C), "packed weights")
    Bp.close()


def test_ahead_switched_off(gm):
    m, n, k = 2100, 1280, 1000
    A, B, C = gi.random_problem(7500, m, n, k, "i16")
    gm.set_option(gm.OPT_SPLIT_AHEAD, 0)
    try:
        got = run(gm, A, B, C, expect_ahead=False)
    finally:
        gm.set_option(gm.OPT_SPLIT_AHEAD, 1)
    assert_same(got, expected(A, B, C), "option off")


@pytest.mark.parametrize("shape", [(2100, 1280, 1001), (1024, 1280, 512), (2100, 64, 512)],
                         ids=["k_not_multiple_of_8", "first_wave_covers_all_panels", "narrow_n_fused"])
def test_ahead_not_taken(gm, shape):
    """Layouts that keep the whole split in front of the GEMM kernel."""
    m, n, k = shape
    A, B, C = gi.random_problem(7600 + k, m, n, k, "i16")
    dA, dB, dC = (torch.from_numpy(x).cuda() for x in (A, B, C))
    counts = counts_of(gm, lambda: gm.gemm_i16(dA, dB, dC))
    assert gm.device_status() == gm.OK
    assert counts["tc_pair_i16_ahead"] == 0, counts
    assert_same(dC.cpu().numpy(), expected(A, B, C), f"{shape}")


def test_ahead_unaligned_A_rows(gm):
    """lda % 8 != 0 (rows of A not 16-byte aligned): the split runs in front."""
    m, n, k = 2100, 1280, 512
    A, B, C = gi.random_problem(7700, m, n, k, "i16")
    Abuf = np.zeros((m, k + 3), np.int16)
    Abuf[:, :k] = A
    dAb, dB, dC = (torch.from_numpy(x).cuda() for x in (Abuf, B, C))
    counts = counts_of(gm, lambda: gm.gemm_i16(dAb[:, :k], dB, dC))
    assert gm.device_status() == gm.OK
    assert counts["tc_pair_i16_ahead"] == 0 and counts["tc_pair_i16"] == 1, counts
    assert_same(dC.cpu().numpy(), expected(A, B, C), "lda = k + 3")
