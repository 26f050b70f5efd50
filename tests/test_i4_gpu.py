"""GPU parity of the int4 GEMM (packed signed nibbles, int32 C) against the oracle, bit for bit.

The int4 path converts both packed operands to E4M3 planes (one byte per value) and runs the SM-pair
kernel on tcgen05.mma kind::f8f6f4.  The cases cover: ragged tiles in every dimension with odd k
and odd n (a spare nibble per row), padded row pitches whose padding bytes must not leak, operands
that are not 16-byte aligned (byte-wise conversion), a C that cannot take 16-byte reductions (the
scratch-and-add path), extreme constant operands, stream-K tails, and reductions long enough that
one exact chunk (2^18 indices at chunk scale 2) fills up with partial sums close to 2^24.
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


@pytest.fixture(params=[1, 2], ids=["chunks_256", "chunks_2^18"])
def chunk_scale(request, gm):
    old = gm.get_option(gm.OPT_TC_CHUNK_SCALE)
    gm.set_option(gm.OPT_TC_CHUNK_SCALE, request.param)
    yield request.param
    gm.set_option(gm.OPT_TC_CHUNK_SCALE, old)


def expected(Ap, Bp, C, k):
    X = C.copy()
    oracle.gemm_i4(Ap, Bp, X, k, nthreads=8)
    return X


def counts_of(gm, fn):
    gm.kernel_timing(True)
    try:
        fn()
        torch.cuda.synchronize()
        return {name: gm.kernel_time(kid)[1] for name, kid in gm.KERNELS}
    finally:
        gm.kernel_timing(False)


def assert_same(got, exp, what=""):
    if not np.array_equal(got, exp):
        bad = np.argwhere(got != exp)
        i, j = bad[0]
        raise AssertionError(f"{what}: {len(bad)} mismatches, first at ({i},{j}): got {got[i, j]} want {exp[i, j]}")


def run(gm, A, B, C, lda=None, ldb=None, ldc=None, pad=0x9B, c_offset=0, expect_direct=None):
    """Pack A (m x k) and B (k x n) with the given byte pitches (padding bytes and spare nibbles
    hold `pad`), run gemm_i4 on the device into columns c_offset .. c_offset+n-1 of an m x ldc
    buffer, check it against the oracle and return the result."""
    m, k = A.shape
    n = B.shape[1]
    lda = lda or (k + 1) // 2
    ldb = ldb or (n + 1) // 2
    ldc = ldc or n + c_offset
    assert ldc >= n + c_offset
    Ap = gi.pack_nibbles(A, ld=lda, pad=pad)
    Bp = gi.pack_nibbles(B, ld=ldb, pad=pad ^ 0xFF)
    Cbuf = gi.uniform_int(4243, (m, ldc), -(1 << 30), 1 << 30, np.int32)
    Cbuf[:, c_offset:c_offset + n] = C
    dA = torch.from_numpy(Ap).cuda()[:, :(k + 1) // 2]
    dB = torch.from_numpy(Bp).cuda()[:, :(n + 1) // 2]
    dCb = torch.from_numpy(Cbuf).cuda()
    counts = counts_of(gm, lambda: gm.gemm_i4(dA, dB, dCb[:, c_offset:c_offset + n], k))
    assert gm.device_status() == gm.OK
    assert counts["tc_pair_i4"] == 1 and counts["convert_i4"] == 1 and counts["split"] == 0, counts
    if expect_direct is not None:
        assert counts["add_i32"] == (0 if expect_direct else 1), counts
    got = dCb.cpu().numpy()
    untouched = np.ones(Cbuf.shape, bool)
    untouched[:, c_offset:c_offset + n] = False
    assert np.array_equal(got[untouched], Cbuf[untouched]), "entries outside the m x n block were written"
    exp = expected(Ap[:, :(k + 1) // 2], Bp[:, :(n + 1) // 2], C, k)
    res = got[:, c_offset:c_offset + n]
    assert_same(res, exp, f"i4 {m}x{n}x{k} lda={lda} ldb={ldb} ldc={ldc}")
    return res


# one tile, ragged tiles with odd k and n, several tiles per pair, k of one partial K block,
# k across exact-chunk and stage boundaries
SHAPES = [(1, 2, 1), (1, 1, 3), (256, 256, 128), (257, 261, 129), (300, 201, 291), (512, 768, 1025),
          (1500, 1100, 513), (100, 2048, 2049), (77, 33, 4099)]


@pytest.mark.parametrize("shape", SHAPES)
def test_i4_shapes(gm, shape):
    m, n, k = shape
    A, B, C = gi.random_problem(8100 + sum(shape), m, n, k, "i4")
    run(gm, A, B, C, expect_direct=n % 4 == 0)  # a dense C of n % 4 != 0 columns takes the scratch path


# (m, n, k, lda, ldb): padded pitches on the 16-byte vector path, then pitches that force the
# byte-wise conversion of A, of B, and of both
LAYOUTS = [(130, 300, 260, 144, 160), (65, 96, 64, 48, 64), (200, 130, 301, 151, 65), (33, 40, 100, 51, 20),
           (90, 70, 90, 45, 35)]


@pytest.mark.parametrize("case", LAYOUTS)
def test_i4_padded_and_unaligned_operands(gm, case):
    m, n, k, lda, ldb = case
    A, B, C = gi.random_problem(8200 + sum(case), m, n, k, "i4")
    run(gm, A, B, C, lda=lda, ldb=ldb)


@pytest.mark.parametrize("ldc,c_offset,direct", [(40, 0, True), (37, 0, False), (38, 0, False), (40, 1, False),
                                                  (44, 4, True)])
def test_i4_c_layouts(gm, ldc, c_offset, direct):
    # C whose base is not 16-byte aligned or whose pitch is not a multiple of 4 elements takes the
    # scratch path: a zeroed int32 array receives the products and one pass adds it into C
    A, B, C = gi.random_problem(8300 + ldc + c_offset, 300, 37, 333, "i4")
    run(gm, A, B, C, ldc=ldc, c_offset=c_offset, expect_direct=direct)


@pytest.mark.parametrize("ab", [(-8, -8), (7, -8), (7, 7), (-8, 7), (-1, 1)])
def test_i4_constant_extremes(gm, ab, chunk_scale):
    a, b = ab
    m, n, k = 300, 260, 5000
    A = np.full((m, k), a, np.int8)
    B = np.full((k, n), b, np.int8)
    C = gi.uniform_int(13, (m, n), -(1 << 30), 1 << 30, np.int32)
    run(gm, A, B, C)


def test_i4_wraps_modulo_2_32(gm):
    A = np.full((64, 4096), -8, np.int8)
    B = np.full((4096, 64), -8, np.int8)
    C = np.full((64, 64), np.iinfo(np.int32).max - 5, np.int32)  # + 262144 wraps past 2^31
    run(gm, A, B, C)


STREAM_K = [(2304, 2304, 1024), (300, 700, 3000), (130, 130, 20000)]


@pytest.mark.parametrize("case", STREAM_K)
def test_i4_stream_k_tails(gm, case, chunk_scale):
    m, n, k = case
    A, B, C = gi.random_problem(8400 + m + n + k, m, n, k, "i4")
    run(gm, A, B, C)


def test_i4_full_chunks_near_2_24(gm, chunk_scale):
    """A reduction of 2*10^7 indices over one 2 x 4 tile: its 156250 K blocks of 128 indices are
    shared out to the pairs (at most 76 on 152 SMs), over 2048 blocks each, so at chunk scale 2
    every share holds one complete chunk of 2048 blocks (2^18 indices).  Row 0 of A is 7
    everywhere and row 1 is -8; column j of B is -8 except -7 at every 32nd index (offset j).
    Every 32 indices then add -1785 (row 0) or +2040 (row 1) to the partial sums, which reach
    about -1.46e7 and +1.67e7 -- within 2^24 = 1.68e7, where every fp32 integer is still exact --
    by the end of a full chunk; sums that lost low bits would fail here."""
    m, n, k = 2, 4, 20_000_000
    A = np.empty((m, k), np.int8)
    A[0] = 7
    A[1] = -8
    B = np.full((k, n), -8, np.int8)
    for j in range(n):
        B[j::32, j] = -7
    C = np.zeros((m, n), np.int32)
    run(gm, A, B, C)


def test_i4_back_to_back_calls_accumulate(gm):
    A, B, C = gi.random_problem(8500, 400, 300, 600, "i4")
    Ap, Bp = gi.pack_nibbles(A), gi.pack_nibbles(B)
    dA, dB, dC = (torch.from_numpy(x).cuda() for x in (Ap, Bp, C))
    for _ in range(3):
        gm.gemm_i4(dA, dB, dC, 600)
    torch.cuda.synchronize()
    exp = C.copy()
    for _ in range(3):
        oracle.gemm_i4(Ap, Bp, exp, 600, nthreads=8)
    assert_same(dC.cpu().numpy(), exp, "three calls")


def test_i4_matches_i8_on_the_same_values(gm):
    # the int4 and int8 device paths give the same C on values in [-8, 7]
    A, B, C = gi.random_problem(8600, 700, 520, 999, "i4")
    dC4 = torch.from_numpy(C.copy()).cuda()
    gm.gemm_i4(torch.from_numpy(gi.pack_nibbles(A)).cuda(), torch.from_numpy(gi.pack_nibbles(B)).cuda(), dC4, 999)
    dC8 = torch.from_numpy(C.copy()).cuda()
    gm.gemm_i8(torch.from_numpy(A).cuda(), torch.from_numpy(B).cuda(), dC8)
    torch.cuda.synchronize()
    assert_same(dC4.cpu().numpy(), dC8.cpu().numpy(), "i4 vs i8")


def test_i4_empty_problems(gm):
    dC = torch.zeros((3, 5), dtype=torch.int32, device="cuda")
    gm.gemm_i4(torch.zeros((3, 1), dtype=torch.uint8, device="cuda"),
               torch.zeros((0, 3), dtype=torch.uint8, device="cuda"), dC, 0)
    torch.cuda.synchronize()
    assert int(dC.abs().sum()) == 0


@pytest.mark.parametrize("case", [(300, 200, 400, None), (77, 131, 257, 80), (1, 6, 3, None)])
def test_i4_packed_weights(gm, case):
    # B converted once to its E4M3 plane (gemmi_pack_b_i4), then used for two different A
    m, n, k, ldb = case
    A, B, C = gi.random_problem(8700 + m, m, n, k, "i4")
    A2 = gi.uniform_int(8701 + m, (m, k), -8, 7, np.int8)
    Bp = gi.pack_nibbles(B, ld=ldb, pad=0x5A)
    packed = gm.pack_b_i4(torch.from_numpy(Bp).cuda()[:, :(n + 1) // 2], n)
    try:
        exp = C.copy()
        for X in (A, A2):
            Ap = gi.pack_nibbles(X)
            dC = torch.from_numpy(exp.copy()).cuda()
            counts = counts_of(gm, lambda: gm.gemm_i4_packed(torch.from_numpy(Ap).cuda(), packed, dC))
            assert counts["tc_pair_i4"] == 1 and counts["convert_i4"] == 1, counts
            assert gm.device_status() == gm.OK
            oracle.gemm_i4(Ap, Bp[:, :(n + 1) // 2], exp, k, nthreads=8)
            assert_same(dC.cpu().numpy(), exp, f"packed i4 {case}")
    finally:
        packed.close()


@pytest.mark.parametrize("case", [(300, 201, 333, None, None), (129, 64, 1000, 520, 40), (2100, 301, 777, 400, 160),
                                  (1024, 64, 256, None, None)])
def test_i4_host_buffers(gm, case):
    # m >= 1024 takes the pipelined host path (row panels through device slots)
    # host arrays with padded byte pitches; the library stages them on the device with aligned pitches
    m, n, k, lda, ldb = case
    A, B, C = gi.random_problem(8800 + m, m, n, k, "i4")
    Ap = gi.pack_nibbles(A, ld=lda, pad=0x3C)[:, :(k + 1) // 2]
    Bp = gi.pack_nibbles(B, ld=ldb, pad=0xC3)[:, :(n + 1) // 2]
    X = C.copy()
    gm.gemm_i4_host(Ap, Bp, X, k)
    exp = C.copy()
    oracle.gemm_i4(np.ascontiguousarray(Ap), np.ascontiguousarray(Bp), exp, k, nthreads=8)
    assert_same(X, exp, f"host i4 {case}")


def test_i4_captured_in_a_cuda_graph_and_on_a_side_stream(gm):
    """Captured calls replay exactly -- the aligned-C path and the scratch path (zeroing and the add
    pass are captured too) -- and calls on a non-default stream order correctly."""
    s = torch.cuda.Stream()
    for n, ldc in ((264, 264), (37, 37)):
        m, k = 300, 333
        A, B, C = gi.random_problem(8900 + n, m, n, k, "i4")
        Ap, Bp = gi.pack_nibbles(A), gi.pack_nibbles(B)
        dA, dB = torch.from_numpy(Ap).cuda(), torch.from_numpy(Bp).cuda()
        dC = torch.from_numpy(C).cuda()
        with torch.cuda.stream(s):
            gm.gemm_i4(dA, dB, torch.from_numpy(C).cuda(), k)  # warm-up outside the capture (workspace growth)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            gm.gemm_i4(dA, dB, dC, k)
        dC.copy_(torch.from_numpy(C).cuda())
        g.replay()
        g.replay()
        torch.cuda.synchronize()
        exp = expected(Ap, Bp, C, k)
        oracle.gemm_i4(Ap, Bp, exp, k)
        assert_same(dC.cpu().numpy(), exp, f"graph x2 n={n}")
        # the same call eagerly on a side stream
        dC2 = torch.from_numpy(C).cuda()
        torch.cuda.synchronize()
        with torch.cuda.stream(s):
            gm.gemm_i4(dA, dB, dC2, k)
        s.synchronize()
        assert_same(dC2.cpu().numpy(), expected(Ap, Bp, C, k), f"side stream n={n}")


def test_i4_binding_rejects_bad_arguments(gm):
    u8 = lambda *shape: torch.zeros(shape, dtype=torch.uint8, device="cuda")  # noqa: E731
    c32 = torch.zeros((4, 6), dtype=torch.int32, device="cuda")
    with pytest.raises(TypeError):
        gm.gemm_i4(torch.zeros((4, 4), dtype=torch.int8, device="cuda"), u8(8, 3), c32, 8)
    with pytest.raises(TypeError):
        gm.gemm_i4(u8(4, 4), u8(8, 3), torch.zeros((4, 6), dtype=torch.int64, device="cuda"), 8)
    with pytest.raises(ValueError):
        gm.gemm_i4(u8(4, 3), u8(8, 3), c32, 8)      # A holds 6 values per row, k = 8
    with pytest.raises(ValueError):
        gm.gemm_i4(u8(4, 4), u8(8, 2), c32, 8)      # B holds 4 values per row, n = 6
    with pytest.raises(ValueError):
        gm.gemm_i4(u8(4, 4), u8(7, 3), c32, 8)      # B has 7 rows, k = 8
    packed = gm.pack_b_i4(u8(8, 3), 6)
    try:
        with pytest.raises(TypeError):               # an int4 handle in the int8 call
            gm.gemm_i8_packed(torch.zeros((4, 8), dtype=torch.int8, device="cuda"), packed, c32)
        with pytest.raises(ValueError):              # A too narrow for the handle's k
            gm.gemm_i4_packed(u8(4, 3), packed, c32)
        # the C ABI itself refuses a handle of another element type
        lib = gm.lib()
        assert lib.gemm_i8_packed(4, torch.zeros((4, 8), dtype=torch.int8, device="cuda").data_ptr(), 8,
                                  packed.handle, c32.data_ptr(), 6, None) == gm.EINVAL
    finally:
        packed.close()
    i8 = gm.pack_b_i8(torch.zeros((8, 6), dtype=torch.int8, device="cuda"))
    try:
        assert gm.lib().gemm_i4_packed(4, u8(4, 4).data_ptr(), 4, i8.handle, c32.data_ptr(), 6, None) == gm.EINVAL
    finally:
        i8.close()
