"""GPU parity of the narrow-n int16 kernel, which reads A raw and splits it into limbs on chip.

Convolutions lowered by im2col give GEMMs with one long and two short
dimensions (the paper's Section 2 workload).  For n <= 64 the library reads A
once, as int16, and converts it in shared memory; these tests check that path
bit for bit against the oracle on ragged shapes, extreme values, both exact-chunk
lengths, the packed-weight entry point and the dispatch rules (which kernel ran
is read back from the library's per-kernel launch counters).
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
    gm.set_option(gm.OPT_FUSED_MAX_N, 64)
    old_small = gm.get_option(gm.OPT_SMALL_MAX_MACS)
    gm.set_option(gm.OPT_SMALL_MAX_MACS, 0)  # small shapes here test this kernel, not the skinny one
    yield gm
    gm.set_option(gm.OPT_FUSED_MAX_N, 64)
    gm.set_option(gm.OPT_SMALL_MAX_MACS, old_small)


@pytest.fixture(params=[1, 2], ids=["chunks_2^23", "chunks_2^24"])
def chunk_scale(request, gm):
    old = gm.get_option(gm.OPT_TC_CHUNK_SCALE)
    gm.set_option(gm.OPT_TC_CHUNK_SCALE, request.param)
    yield request.param
    gm.set_option(gm.OPT_TC_CHUNK_SCALE, old)


def expected(A, B, C):
    X = C.copy()
    oracle.gemm(A, B, X, nthreads=8)
    return X


def launches(gm, fn):
    """Runs fn() with kernel timing on; returns {kernel name: launches}."""
    gm.kernel_timing(True)
    try:
        fn()
        torch.cuda.synchronize()
        return {name: gm.kernel_time(kid)[1] for name, kid in gm.KERNELS}
    finally:
        gm.kernel_timing(False)


def device_a(A, seed=0):
    """A on the device with a row pitch (lda) that is a multiple of 8, as the fused kernel's TMA
    reads need; the padding columns hold random values that must not leak into C."""
    m, k = A.shape
    lda = -(-k // 8) * 8
    if lda == k:
        return torch.from_numpy(np.ascontiguousarray(A)).cuda()
    Apad = gi.uniform_int(seed + 5000, (m, lda), -32768, 32767, np.int16)
    Apad[:, :k] = A
    return torch.from_numpy(Apad).cuda()[:, :k]


def run(gm, A, B, C, expect_fused=True):
    dA = device_a(A)
    dB, dC = (torch.from_numpy(np.ascontiguousarray(x)).cuda() for x in (B, C))
    counts = launches(gm, lambda: gm.gemm_i16(dA, dB, dC))
    assert gm.device_status() == gm.OK
    assert (counts["fused_i16"] == 1) == expect_fused, counts
    assert counts["tc_i16"] + counts["tc_pair_i16"] + counts["tc_pair_i16_ahead"] == (0 if expect_fused else 1), counts
    return dC.cpu().numpy()


def assert_same(got, exp, what=""):
    if not np.array_equal(got, exp):
        bad = np.argwhere(got != exp)
        i, j = bad[0]
        raise AssertionError(f"{what}: {len(bad)} mismatches, first at ({i},{j}): got {got[i, j]} want {exp[i, j]}")


# m spans several 128-row tiles with a ragged tail; k covers one partial K block, exact multiples
# of the 64-wide K block, the conv's 576, and runs longer than one exact chunk (512 / 1024).
SHAPES = [(17, 1, 1), (17, 64, 1), (129, 64, 576), (300, 33, 100), (1000, 64, 576), (513, 7, 1025),
          (250, 64, 2049), (4000, 48, 577), (128, 63, 64), (20000, 64, 576), (257, 16, 4096)]


@pytest.mark.parametrize("shape", SHAPES)
def test_fused_shapes(gm, shape):
    m, n, k = shape
    A, B, C = gi.random_problem(700 + sum(shape), m, n, k, "i16")
    assert_same(run(gm, A, B, C), expected(A, B, C), f"fused {shape}")


EXTREMES = [(-32768, -32768), (32767, 32767), (32640, 32640), (32641, 32641), (-32641, 32641), (-129, 32767),
            (127, -128), (128, 255)]


@pytest.mark.parametrize("ab", EXTREMES)
def test_fused_constant_extremes(gm, ab, chunk_scale):
    a, b = ab
    m, n, k = 300, 64, 2600
    A = np.full((m, k), a, np.int16)
    B = np.full((k, n), b, np.int16)
    C = gi.uniform_int(11, (m, n), -(1 << 40), 1 << 40, np.int64)
    assert_same(run(gm, A, B, C), expected(A, B, C), f"constant {ab}, chunk scale {chunk_scale}")


def test_fused_every_int16_value_of_A(gm, chunk_scale):
    # all 65536 int16 values appear in A, so the on-chip split meets every bit pattern
    m, k, n = 256, 256, 64
    A = (np.arange(m * k, dtype=np.int64) - 32768).astype(np.int16).reshape(m, k)
    A = A[gi.uniform_int(12, (m,), 0, m - 1, np.int64).argsort()]  # shuffle rows
    B = gi.uniform_int(13, (k, n), -32768, 32767, np.int16)
    C = np.zeros((m, n), np.int64)
    assert_same(run(gm, A, B, C), expected(A, B, C), "every int16 value")


def test_fused_matches_split_path(gm):
    # the same call with the fused kernel switched off runs split + tcgen05 GEMM
    A, B, C = gi.random_problem(720, 777, 64, 700, "i16")
    got_fused = run(gm, A, B, C, expect_fused=True)
    gm.set_option(gm.OPT_FUSED_MAX_N, 0)
    try:
        got_split = run(gm, A, B, C, expect_fused=False)
    finally:
        gm.set_option(gm.OPT_FUSED_MAX_N, 64)
    assert_same(got_fused, got_split, "fused vs split")
    assert_same(got_fused, expected(A, B, C), "fused vs oracle")


def test_fused_wider_n_via_option(gm):
    # with the limit raised, n = 200 runs as four 64-column tiles (the last one ragged)
    A, B, C = gi.random_problem(721, 333, 200, 300, "i16")
    gm.set_option(gm.OPT_FUSED_MAX_N, 256)
    try:
        got = run(gm, A, B, C, expect_fused=True)
    finally:
        gm.set_option(gm.OPT_FUSED_MAX_N, 64)
    assert_same(got, expected(A, B, C), "fused n=200")


def test_fused_dispatch_rules(gm):
    A, B, C = gi.random_problem(722, 200, 64, 96, "i16")
    # n above the limit: the general path
    A2, B2, C2 = gi.random_problem(723, 200, 65, 96, "i16")
    assert_same(run(gm, A2, B2, C2, expect_fused=False), expected(A2, B2, C2), "n=65")
    # lda not a multiple of 8: TMA cannot read A, the general path
    Apad = np.zeros((200, 99), np.int16)
    Apad[:, :96] = A
    dA = torch.from_numpy(Apad).cuda()[:, :96]
    dB, dC = torch.from_numpy(B).cuda(), torch.from_numpy(C).cuda()
    counts = launches(gm, lambda: gm.gemm_i16(dA, dB, dC))
    assert counts["fused_i16"] == 0 and counts["tc_i16"] + counts["tc_pair_i16"] + counts["tc_pair_i16_ahead"] == 1, counts
    assert_same(dC.cpu().numpy(), expected(A, B, C), "lda=99")
    # lda a multiple of 8 with padding: fused
    Apad = np.zeros((200, 104), np.int16)
    Apad[:, :96] = A
    dA = torch.from_numpy(Apad).cuda()[:, :96]
    dC = torch.from_numpy(C).cuda()
    counts = launches(gm, lambda: gm.gemm_i16(dA, dB, dC))
    assert counts["fused_i16"] == 1, counts
    assert_same(dC.cpu().numpy(), expected(A, B, C), "lda=104")


# ldc odd: element-wise atomic adds; ldc even: one bulk reduction per row (n < 64 or ldc > n)
@pytest.mark.parametrize("n,ldc", [(40, 45), (40, 48), (64, 72), (33, 34)])
def test_fused_padded_c(gm, n, ldc):
    A, B, C = gi.random_problem(724 + ldc, 300, n, 577, "i16")
    Cpad = gi.uniform_int(725, (300, ldc), -(1 << 50), 1 << 50, np.int64)
    Cpad[:, :n] = C
    dA, dB = device_a(A), torch.from_numpy(B).cuda()
    dCp = torch.from_numpy(Cpad).cuda()
    counts = launches(gm, lambda: gm.gemm_i16(dA, dB, dCp[:, :n]))
    assert counts["fused_i16"] == 1, counts
    got = dCp.cpu().numpy()
    assert_same(got[:, :n], expected(A, B, C), f"ldc={ldc}")
    assert np.array_equal(got[:, n:], Cpad[:, n:]), "columns beyond n were written"


def test_fused_c_not_16_byte_aligned(gm):
    # C starts 8 bytes into a buffer: row segments cannot go out as 16-byte bulk reductions,
    # the kernel adds them element by element
    A, B, C = gi.random_problem(728, 400, 64, 300, "i16")
    Cbuf = gi.uniform_int(729, (400, 66), -(1 << 50), 1 << 50, np.int64)
    Cbuf[:, 1:65] = C
    dA, dB = device_a(A), torch.from_numpy(B).cuda()
    dCb = torch.from_numpy(Cbuf).cuda()
    view = dCb[:, 1:65]
    assert view.data_ptr() % 16 == 8
    counts = launches(gm, lambda: gm.gemm_i16(dA, dB, view))
    assert counts["fused_i16"] == 1, counts
    got = dCb.cpu().numpy()
    assert_same(got[:, 1:65], expected(A, B, C), "C offset by 8 bytes")
    assert np.array_equal(got[:, [0, 65]], Cbuf[:, [0, 65]]), "columns outside C were written"


def test_fused_with_packed_weights(gm):
    A, B, C = gi.random_problem(726, 1500, 64, 576, "i16")
    dB = torch.from_numpy(B).cuda()
    packed = gm.pack_b_i16(dB)
    try:
        dA, dC = device_a(A), torch.from_numpy(C).cuda()
        counts = launches(gm, lambda: gm.gemm_i16_packed(dA, packed, dC))
        assert counts["fused_i16"] == 1 and counts["split"] == 0, counts
        assert gm.device_status() == gm.OK
        assert_same(dC.cpu().numpy(), expected(A, B, C), "packed")
    finally:
        packed.close()


def test_fused_conv_workload_every_element(gm):
    """The im2col workload (m = 100352, n = 64, k = 576) through the fused kernel: every element of C
    against the oracle (all host cores), plus row and column sums as an extra check."""
    w = gi.WORKLOADS["conv3x3_im2col"]
    A, B, C = gi.make_inputs(w)
    dA, dB, dC = (torch.from_numpy(x).cuda() for x in (A, B, C))
    counts = launches(gm, lambda: gm.gemm_i16(dA, dB, dC))
    assert counts["fused_i16"] == 1, counts
    got = dC.cpu().numpy()
    exp = C.copy()
    oracle.gemm(A, B, exp, nthreads=oracle.host_cores())
    assert_same(got, exp, "conv workload, all outputs")
    # every output: row and column sums (mod 2^64)
    with np.errstate(over="ignore"):
        a64, b64 = A.astype(np.int64), B.astype(np.int64)
        exp_rows = C.sum(axis=1, dtype=np.int64) + a64 @ b64.sum(axis=1, dtype=np.int64)
        exp_cols = C.sum(axis=0, dtype=np.int64) + a64.sum(axis=0, dtype=np.int64) @ b64
        assert np.array_equal(got.sum(axis=1, dtype=np.int64), exp_rows)
        assert np.array_equal(got.sum(axis=0, dtype=np.int64), exp_cols)
