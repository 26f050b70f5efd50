"""GPU parity of the SM-pair tensor-core kernels (tcgen05 cta_group::2) against the oracle, bit for bit.

The pair kernels add each finished tile into C with bulk reductions, and the two SMs of an int16
tile add their weighted halves independently; these tests cover what that changes: ragged tiles
whose last row segment is not a whole number of 16-byte units (element-wise tail), C with a padded
row pitch (columns past n untouched), the persistent tile loop (more tiles than pairs), both
exact-chunk lengths, extreme constant operands, and the dispatch rule (a C that cannot take 16-byte
reductions goes to the single-SM kernel).  Which kernel ran is read back from the library's
per-kernel launch counters.
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
    gm.set_option(gm.OPT_TC_PAIR, 1)
    gm.set_option(gm.OPT_SKINNY_MAX_M, 0)   # small m also runs on the tensor cores here
    gm.set_option(gm.OPT_FUSED_MAX_N, 0)    # and narrow n
    yield gm
    gm.set_option(gm.OPT_TC_PAIR, 1)
    gm.set_option(gm.OPT_SKINNY_MAX_M, 16)
    gm.set_option(gm.OPT_FUSED_MAX_N, 64)


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


def counts_of(gm, fn):
    gm.kernel_timing(True)
    try:
        fn()
        torch.cuda.synchronize()
        return {name: gm.kernel_time(kid)[1] for name, kid in gm.KERNELS}
    finally:
        gm.kernel_timing(False)


def run(gm, A, B, C, ldc=None, expect_pair=True):
    """C += A*B on the device, C held with row pitch ldc (>= n); returns the whole padded buffer."""
    kind = "i16" if A.dtype == np.int16 else "i8"
    m, n = C.shape
    ldc = ldc or n
    Cbuf = gi.uniform_int(4242, (m, ldc), -(1 << 30), 1 << 30, C.dtype)
    Cbuf[:, :n] = C
    dA, dB = (torch.from_numpy(np.ascontiguousarray(x)).cuda() for x in (A, B))
    dCb = torch.from_numpy(Cbuf).cuda()
    fn = gm.gemm_i16 if kind == "i16" else gm.gemm_i8
    counts = counts_of(gm, lambda: fn(dA, dB, dCb[:, :n]))
    assert gm.device_status() == gm.OK
    pair_name, single_name = (("tc_pair_i16", "tc_i16") if kind == "i16" else ("tc_pair_i8", "tc_i8"))
    pair_launches = counts[pair_name] + (counts["tc_pair_i16_ahead"] if kind == "i16" else 0)
    assert pair_launches == (1 if expect_pair else 0), counts
    assert counts[single_name] == (0 if expect_pair else 1), counts
    got = dCb.cpu().numpy()
    assert np.array_equal(got[:, n:], Cbuf[:, n:]), "columns beyond n were written"
    return got[:, :n]


def assert_same(got, exp, what=""):
    if not np.array_equal(got, exp):
        bad = np.argwhere(got != exp)
        i, j = bad[0]
        raise AssertionError(f"{what}: {len(bad)} mismatches, first at ({i},{j}): got {got[i, j]} want {exp[i, j]}")


# m, n, k: one tile, ragged tiles in every dimension, several tiles per pair (persistent loop),
# k of one partial K block, exact chunk multiples and one past them
SHAPES_I16 = [(1, 2, 1), (128, 128, 64), (129, 130, 65), (300, 200, 290), (256, 384, 1025), (1000, 640, 513),
              (2048, 1536, 96), (64, 1000, 2049), (700, 256, 4096)]


@pytest.mark.parametrize("shape", SHAPES_I16)
def test_pair_i16_shapes(gm, shape):
    m, n, k = shape
    A, B, C = gi.random_problem(5100 + sum(shape), m, n, k, "i16")
    assert_same(run(gm, A, B, C), expected(A, B, C), f"pair i16 {shape}")


SHAPES_I8 = [(1, 4, 1), (256, 256, 64), (257, 260, 65), (300, 200, 290), (512, 768, 1025), (1500, 1100, 513),
             (100, 2048, 2049)]


@pytest.mark.parametrize("shape", SHAPES_I8)
def test_pair_i8_shapes(gm, shape):
    m, n, k = shape
    A, B, C = gi.random_problem(5200 + sum(shape), m, n, k, "i8")
    assert_same(run(gm, A, B, C), expected(A, B, C), f"pair i8 {shape}")


# n whose last 16-byte unit of a row segment is partial: int64 with n odd, int32 with n % 4 != 0;
# ldc padded so C still takes 16-byte reductions
@pytest.mark.parametrize("kind,n,ldc", [("i16", 37, 38), ("i16", 129, 130), ("i16", 255, 258),
                                        ("i8", 37, 40), ("i8", 130, 132), ("i8", 259, 260)])
def test_pair_ragged_row_tail(gm, kind, n, ldc):
    A, B, C = gi.random_problem(5300 + n, 300, n, 333, kind)
    assert_same(run(gm, A, B, C, ldc=ldc), expected(A, B, C), f"{kind} n={n} ldc={ldc}")


EXTREMES = [(-32768, -32768), (32767, 32767), (-32768, 32767), (32640, 32641), (-129, 128)]


@pytest.mark.parametrize("ab", EXTREMES)
def test_pair_i16_constant_extremes(gm, ab, chunk_scale):
    a, b = ab
    m, n, k = 200, 136, 2600
    A = np.full((m, k), a, np.int16)
    B = np.full((k, n), b, np.int16)
    C = gi.uniform_int(11, (m, n), -(1 << 40), 1 << 40, np.int64)
    assert_same(run(gm, A, B, C), expected(A, B, C), f"constant {ab}, chunk scale {chunk_scale}")


@pytest.mark.parametrize("ab", [(-128, -128), (127, 127), (-128, 127)])
def test_pair_i8_constant_extremes(gm, ab, chunk_scale):
    a, b = ab
    m, n, k = 300, 260, 3000
    A = np.full((m, k), a, np.int8)
    B = np.full((k, n), b, np.int8)
    C = gi.uniform_int(12, (m, n), -(1 << 30), 1 << 30, np.int32)
    assert_same(run(gm, A, B, C), expected(A, B, C), f"constant {ab}, chunk scale {chunk_scale}")


def test_pair_i16_wraps_modulo_2_64(gm):
    # C near the int64 limits: the sums wrap exactly as the oracle's unsigned arithmetic does
    A = np.full((130, 5000), -32768, np.int16)
    B = np.full((5000, 64), -32768, np.int16)
    C = np.full((130, 64), np.iinfo(np.int64).max - 5, np.int64)
    assert_same(run(gm, A, B, C), expected(A, B, C), "wrap")


def test_pair_every_int16_value(gm, chunk_scale):
    m, k, n = 256, 256, 128
    A = (np.arange(m * k, dtype=np.int64) - 32768).astype(np.int16).reshape(m, k)
    B = A.T.copy()[:, :n]
    C = np.zeros((m, n), np.int64)
    assert_same(run(gm, A, B, C), expected(A, B, C), "every int16 value")


def test_pair_matches_single_sm_kernel(gm):
    A, B, C = gi.random_problem(5400, 777, 520, 1500, "i16")
    got_pair = run(gm, A, B, C, expect_pair=True)
    gm.set_option(gm.OPT_TC_PAIR, 0)
    try:
        got_single = run(gm, A, B, C, expect_pair=False)
    finally:
        gm.set_option(gm.OPT_TC_PAIR, 1)
    assert_same(got_pair, got_single, "pair vs single")
    assert_same(got_pair, expected(A, B, C), "pair vs oracle")


def test_pair_dispatch_needs_16_byte_c(gm):
    # ldc * 8 not a multiple of 16: the single-SM kernel runs
    A, B, C = gi.random_problem(5500, 200, 64, 96, "i16")
    assert_same(run(gm, A, B, C, ldc=65, expect_pair=False), expected(A, B, C), "ldc=65")
    # C starting 8 bytes into its buffer: the single-SM kernel runs
    Cbuf = gi.uniform_int(5501, (200, 66), -(1 << 50), 1 << 50, np.int64)
    Cbuf[:, 1:65] = C
    dA, dB = torch.from_numpy(A).cuda(), torch.from_numpy(B).cuda()
    dCb = torch.from_numpy(Cbuf).cuda()
    counts = counts_of(gm, lambda: gm.gemm_i16(dA, dB, dCb[:, 1:65]))
    assert counts["tc_pair_i16"] + counts["tc_pair_i16_ahead"] == 0 and counts["tc_i16"] == 1, counts
    got = dCb.cpu().numpy()
    assert_same(got[:, 1:65], expected(A, B, C), "C offset by 8 bytes")
    assert np.array_equal(got[:, [0, 65]], Cbuf[:, [0, 65]])


def test_pair_packed_weights(gm):
    A, B, C = gi.random_problem(5600, 900, 320, 700, "i16")
    dB = torch.from_numpy(B).cuda()
    packed = gm.pack_b_i16(dB)
    try:
        dA, dC = torch.from_numpy(A).cuda(), torch.from_numpy(C).cuda()
        counts = counts_of(gm, lambda: gm.gemm_i16_packed(dA, packed, dC))
        assert counts["tc_pair_i16"] + counts["tc_pair_i16_ahead"] == 1, counts
        assert gm.device_status() == gm.OK
        assert_same(dC.cpu().numpy(), expected(A, B, C), "packed")
    finally:
        packed.close()


def test_pair_back_to_back_calls_accumulate(gm):
    # three calls into the same C: every call's reductions land before the next reads nothing
    # (the kernels never read C), so the sum of the three products must come out
    A, B, C = gi.random_problem(5700, 400, 300, 600, "i16")
    dA, dB, dC = (torch.from_numpy(x).cuda() for x in (A, B, C))
    for _ in range(3):
        gm.gemm_i16(dA, dB, dC)
    torch.cuda.synchronize()
    exp = C.copy()
    for _ in range(3):
        oracle.gemm(A, B, exp, nthreads=8)
    assert_same(dC.cpu().numpy(), exp, "three calls")


# Stream-K tails: more tiles than pairs with a partial last wave (its K blocks are shared out, so
# segments start and end inside tiles), and fewer tiles than pairs (every tile split along K)
STREAM_K = [("i16", 1408, 896, 2048), ("i16", 600, 300, 4096), ("i16", 130, 130, 1100), ("i8", 2304, 2304, 1024),
            ("i8", 300, 700, 3000)]


@pytest.mark.parametrize("case", STREAM_K)
def test_pair_stream_k_tails(gm, case, chunk_scale):
    kind, m, n, k = case
    A, B, C = gi.random_problem(5800 + m + n + k, m, n, k, kind)
    assert_same(run(gm, A, B, C), expected(A, B, C), f"stream-K {case}, chunk scale {chunk_scale}")


# long reductions over few tiles: every pair's stream-K share starts and ends inside a tile and
# crosses exact-chunk boundaries at arbitrary offsets
@pytest.mark.parametrize("kind,m,n,k", [("i16", 130, 130, 20000), ("i8", 300, 260, 30011), ("i16", 1, 2, 65537)])
def test_pair_long_reduction_stream_k(gm, kind, m, n, k, chunk_scale):
    A, B, C = gi.random_problem(5900 + k, m, n, k, kind)
    assert_same(run(gm, A, B, C), expected(A, B, C), f"{kind} {m}x{n}x{k}, chunk scale {chunk_scale}")
