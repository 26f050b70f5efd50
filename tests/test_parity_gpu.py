"""GPU parity: the CUDA path through the C ABI against the CPU oracle, bit for bit.

Expected values always come from the oracle (oracle/) run on the same seeded
inputs (gemm_inputs.py); nothing here is produced by the CUDA path itself.
The five full-size workloads are compared on every output element; the
int4 workload on sampled rows plus a row-sum/column-sum identity that covers
every output:  sum_j C[i,j] = A[i,:] . (B 1),  sum_i C[i,j] = (1^T A) . B[:,j].
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
    gm.lib()  # raises if the library was not built
    gm.set_option(gm.OPT_SKINNY_MAX_M, 16)
    gm.set_option(gm.OPT_SKINNY_KSPLIT, 0)
    yield gm
    gm.set_option(gm.OPT_SKINNY_MAX_M, 16)
    gm.set_option(gm.OPT_SKINNY_KSPLIT, 0)


def expected(A, B, C, threads=8):
    X = C.copy()
    oracle.gemm(A, B, X, nthreads=threads)
    return X


def run_gpu(gm, A, B, C, kind=None):
    kind = kind or ("i16" if A.dtype == np.int16 else "i8")
    if kind == "i4":  # int4 values in int8 arrays, stored packed for the device
        dA, dB, dC = (torch.from_numpy(x).cuda() for x in (gi.pack_nibbles(A), gi.pack_nibbles(B), C))
        gm.gemm_i4(dA, dB, dC, A.shape[1])
        torch.cuda.synchronize()
        assert gm.device_status() == gm.OK
        return dC.cpu().numpy()
    dA, dB, dC = (torch.from_numpy(np.ascontiguousarray(x)).cuda() for x in (A, B, C))
    (gm.gemm_i16 if kind == "i16" else gm.gemm_i8)(dA, dB, dC)
    torch.cuda.synchronize()
    assert gm.device_status() == gm.OK
    return dC.cpu().numpy()


def assert_same(got, exp, what=""):
    if not np.array_equal(got, exp):
        bad = np.argwhere(got != exp)
        i, j = bad[0]
        raise AssertionError(f"{what}: {len(bad)} mismatches, first at ({i},{j}): got {got[i, j]} want {exp[i, j]}")


# ------------------------------------------------------------------ small and ragged shapes, full comparison
SHAPES_I16 = [
    (1, 1, 1), (2, 3, 5), (17, 33, 1), (128, 128, 64), (129, 127, 65), (300, 200, 290),
    (256, 384, 513), (200, 130, 1000), (130, 260, 2049), (512, 384, 290), (64, 513, 700),
]


@pytest.mark.parametrize("shape", SHAPES_I16)
def test_i16_shapes(gm, shape):
    m, n, k = shape
    A, B, C = gi.random_problem(100 + sum(shape), m, n, k, "i16")
    assert_same(run_gpu(gm, A, B, C), expected(A, B, C), f"i16 {shape}")


@pytest.mark.parametrize("shape", [(1, 1, 1), (20, 40, 60), (129, 130, 131), (256, 256, 1025), (300, 77, 2100)])
def test_i8_shapes(gm, shape):
    m, n, k = shape
    A, B, C = gi.random_problem(200 + sum(shape), m, n, k, "i8")
    assert_same(run_gpu(gm, A, B, C), expected(A, B, C), f"i8 {shape}")


@pytest.fixture(params=["dispatch", "tensor_cores"])
def path(request, gm):
    """The library's own choice of kernel, and the tensor-core path forced for shapes that the
    small-problem rule would give to the skinny kernel."""
    old = gm.get_option(gm.OPT_SMALL_MAX_MACS)
    if request.param == "tensor_cores":
        gm.set_option(gm.OPT_SMALL_MAX_MACS, 0)
    yield request.param
    gm.set_option(gm.OPT_SMALL_MAX_MACS, old)


@pytest.mark.parametrize("k", [511, 512, 513, 1023, 1024, 1025, 4096])
def test_i16_chunk_boundaries(gm, k, path):
    A, B, C = gi.random_problem(300 + k, 160, 136, k, "i16")
    assert_same(run_gpu(gm, A, B, C), expected(A, B, C), f"k={k}")


# ------------------------------------------------------------------ extreme and adversarial values
# 32640 has limbs (h, l) = (128, -128): every limb product is +-2^14, the largest possible.
# +-32641 have limbs (128, -127) / (-128, 127): limb products 16384, -16256, 16129 -- odd and
# within 2% of the largest, so a chunk's partial sums run up to just below its bound with the
# low bit changing at every step, where any loss of precision in the accumulation would show.
EXTREMES = [(-32768, -32768), (32767, -32768), (32767, 32767), (32640, 32640), (-1, -1), (32640, -32768),
            (-129, 32767), (32641, 32641), (-32641, 32641), (-32641, -32641)]


@pytest.fixture(params=[1, 2], ids=["chunks_2^23", "chunks_2^24"])
def chunk_scale(request, gm):
    old = gm.get_option(gm.OPT_TC_CHUNK_SCALE)
    gm.set_option(gm.OPT_TC_CHUNK_SCALE, request.param)
    yield request.param
    gm.set_option(gm.OPT_TC_CHUNK_SCALE, old)


@pytest.mark.parametrize("ab", EXTREMES)
@pytest.mark.parametrize("m", [8, 200])
def test_i16_constant_extremes(gm, ab, m, chunk_scale, path):
    a, b = ab
    n, k = 136, 2600
    A = np.full((m, k), a, np.int16)
    B = np.full((k, n), b, np.int16)
    C = gi.uniform_int(9, (m, n), -(1 << 40), 1 << 40, np.int64)
    assert_same(run_gpu(gm, A, B, C), expected(A, B, C), f"constant {ab} chunk scale {chunk_scale}")


@pytest.mark.parametrize("m", [8, 160])
def test_i16_near_fp32_exactness_limit(gm, m, chunk_scale, path):
    """Limb sums pushed toward the largest magnitudes a chunk allows, with odd low bits.

    32640 = 256*128 - 128 has limbs (h, l) = (128, -128): every limb product is
    +-2^14, the most a product can be.  Mixing in values with low bits set makes
    the partial sums large and odd, where a lossy accumulation would show.
    """
    n, k = 136, 2048
    base = np.where((np.arange(k) % 7) == 3, -32767, 32640).astype(np.int16)
    A = np.tile(base, (m, 1))
    A[:, ::13] = 32767
    B = np.tile(base[:, None], (1, n)).astype(np.int16)
    B[::11, :] = -32768
    B[5::17, ::3] = 255
    C = np.zeros((m, n), np.int64)
    assert_same(run_gpu(gm, A, B, C), expected(A, B, C), "adversarial")


def test_i8_extremes(gm, chunk_scale):
    for a, b in ((-128, -128), (127, -128), (127, 127), (-127, -127)):
        A = np.full((140, 3000), a, np.int8)
        B = np.full((3000, 136), b, np.int8)
        C = gi.uniform_int(3, (140, 136), -(1 << 30), 1 << 30, np.int32)
        assert_same(run_gpu(gm, A, B, C), expected(A, B, C), f"i8 constant {(a, b)}")


def test_wraparound_mod_2_64(gm):
    A = np.full((130, 4), 32767, np.int16)
    B = np.full((4, 130), 32767, np.int16)
    C = np.full((130, 130), np.iinfo(np.int64).max - 5, np.int64)
    assert_same(run_gpu(gm, A, B, C), expected(A, B, C), "wrap")


# ------------------------------------------------------------------ layouts: padding, odd leading dimensions
@pytest.mark.parametrize("pads", [(0, 0, 0), (3, 5, 7), (8, 8, 2), (1, 0, 1)])
@pytest.mark.parametrize("m", [5, 150])
def test_i16_leading_dimensions(gm, pads, m):
    pa, pb, pc = pads
    n, k = 140, 333
    A, B, C = gi.random_problem(400 + m + sum(pads), m, n, k, "i16")
    exp = expected(A, B, C)
    Ap = torch.full((m, k + pa), 12345, dtype=torch.int16)
    Bp = torch.full((k, n + pb), -777, dtype=torch.int16)
    Cp = torch.full((m, n + pc), -424242, dtype=torch.int64)
    Ap[:, :k] = torch.from_numpy(A)
    Bp[:, :n] = torch.from_numpy(B)
    Cp[:, :n] = torch.from_numpy(C)
    dA, dB, dC = Ap.cuda(), Bp.cuda(), Cp.cuda()
    gm.gemm_i16(dA[:, :k], dB[:, :n], dC[:, :n])
    torch.cuda.synchronize()
    out = dC.cpu().numpy()
    assert_same(out[:, :n], exp, f"padded {pads}")
    assert (out[:, n:] == -424242).all(), "padding of C was written"


def test_i8_leading_dimensions(gm):
    m, n, k = 150, 131, 517
    A, B, C = gi.random_problem(77, m, n, k, "i8")
    exp = expected(A, B, C)
    Ap = torch.zeros((m, k + 3), dtype=torch.int8)
    Bp = torch.zeros((k, n + 5), dtype=torch.int8)
    Cp = torch.full((m, n + 1), 99, dtype=torch.int32)
    Ap[:, :k], Bp[:, :n], Cp[:, :n] = torch.from_numpy(A), torch.from_numpy(B), torch.from_numpy(C)
    dA, dB, dC = Ap.cuda(), Bp.cuda(), Cp.cuda()
    gm.gemm_i8(dA[:, :k], dB[:, :n], dC[:, :n])
    torch.cuda.synchronize()
    out = dC.cpu().numpy()
    assert_same(out[:, :n], exp, "i8 padded")
    assert (out[:, n:] == 99).all()


# ------------------------------------------------------------------ skinny-M path
@pytest.mark.parametrize("m", [1, 3, 8, 9, 16])
@pytest.mark.parametrize("nk", [(100, 300), (4096, 1000), (33, 4097)])
def test_skinny_shapes(gm, m, nk):
    n, k = nk
    A, B, C = gi.random_problem(500 + m + n + k, m, n, k, "i16")
    assert_same(run_gpu(gm, A, B, C), expected(A, B, C), f"skinny m={m} n={n} k={k}")


@pytest.mark.parametrize("ksplit", [1, 2, 5, 64])
def test_skinny_ksplit(gm, ksplit):
    gm.set_option(gm.OPT_SKINNY_KSPLIT, ksplit)
    try:
        A, B, C = gi.random_problem(600 + ksplit, 8, 1000, 3000, "i16")
        assert_same(run_gpu(gm, A, B, C), expected(A, B, C), f"ksplit={ksplit}")
    finally:
        gm.set_option(gm.OPT_SKINNY_KSPLIT, 0)


def test_main_kernel_on_small_m(gm):
    """The tcgen05 path on m <= 16 (skinny path switched off)."""
    gm.set_option(gm.OPT_SKINNY_MAX_M, 0)
    try:
        for m in (1, 8, 16):
            A, B, C = gi.random_problem(700 + m, m, 260, 700, "i16")
            assert_same(run_gpu(gm, A, B, C), expected(A, B, C), f"tc m={m}")
    finally:
        gm.set_option(gm.OPT_SKINNY_MAX_M, 16)


def test_skinny_unaligned_B(gm):
    m, n, k = 8, 203, 900
    A, B, C = gi.random_problem(801, m, n, k, "i16")
    exp = expected(A, B, C)
    Bp = torch.zeros((k, n + 1), dtype=torch.int16)  # row pitch 204 elements = 408 bytes: not 16-aligned
    Bp[:, :n] = torch.from_numpy(B)
    dA, dB, dC = torch.from_numpy(A).cuda(), Bp.cuda(), torch.from_numpy(C).cuda()
    gm.gemm_i16(dA, dB[:, :n], dC)
    torch.cuda.synchronize()
    assert_same(dC.cpu().numpy(), exp, "skinny unaligned B")


# the CTA's slice of A is bulk-copied when A's rows are 16-byte aligned and k % 8 == 0, and
# loaded element by element otherwise; both with padded leading dimensions and ragged k ranges
@pytest.mark.parametrize("m,k,lda", [(8, 4096, 4096), (5, 1000, 1008), (16, 2040, 2048), (3, 1000, 1001),
                                     (8, 999, 1000), (13, 96, 104)])
def test_skinny_a_slice_paths(gm, m, k, lda):
    n = 700
    A, B, C = gi.random_problem(805 + m + k + lda, m, n, k, "i16")
    Ap = torch.full((m, lda), 31000, dtype=torch.int16)
    Ap[:, :k] = torch.from_numpy(A)
    dA, dB, dC = Ap.cuda(), torch.from_numpy(B).cuda(), torch.from_numpy(C).cuda()
    gm.gemm_i16(dA[:, :k], dB, dC)
    torch.cuda.synchronize()
    assert gm.device_status() == gm.OK
    assert_same(dC.cpu().numpy(), expected(A, B, C), f"skinny m={m} k={k} lda={lda}")


def _kernel_counts(gm, fn):
    gm.kernel_timing(True)
    try:
        fn()
        torch.cuda.synchronize()
        return {name: gm.kernel_time(kid)[1] for name, kid in gm.KERNELS}
    finally:
        gm.kernel_timing(False)


# small problems (m <= 256, m*n*k <= 2^28 by default) run the skinny kernel with one grid row per
# 16 rows of A: the last group ragged, several column blocks and reduction splits
@pytest.mark.parametrize("m,n,k", [(17, 64, 64), (24, 300, 1000), (100, 513, 576), (255, 256, 256), (256, 256, 256),
                                   (200, 40, 4000)])
def test_skinny_row_groups(gm, m, n, k):
    A, B, C = gi.random_problem(830 + m + n + k, m, n, k, "i16")
    dA, dB, dC = (torch.from_numpy(x).cuda() for x in (A, B, C))
    counts = _kernel_counts(gm, lambda: gm.gemm_i16(dA, dB, dC))
    assert gm.device_status() == gm.OK
    assert counts["skinny"] == 1 and counts["split"] == 0, counts
    assert_same(dC.cpu().numpy(), expected(A, B, C), f"skinny row groups {m}x{n}x{k}")


@pytest.mark.parametrize("m,n,k,skinny", [(256, 1024, 1024, True), (255, 1000, 1050, True), (256, 1024, 1025, False)])
def test_small_problem_limit(gm, m, n, k, skinny):
    # at the default limit of 2^28 multiply-adds: 256 x 1024 x 1024 is the largest 256-row problem
    # the skinny kernel takes (16 row groups x 2 column blocks x 4 reduction ranges of 8 stages)
    assert gm.get_option(gm.OPT_SMALL_MAX_MACS) == 1 << 28
    A, B, C = gi.random_problem(860 + m + n + k, m, n, k, "i16")
    dA, dB, dC = (torch.from_numpy(x).cuda() for x in (A, B, C))
    counts = _kernel_counts(gm, lambda: gm.gemm_i16(dA, dB, dC))
    assert gm.device_status() == gm.OK
    if skinny:
        assert counts["skinny"] == 1 and counts["split"] == 0, counts
    else:
        assert counts["skinny"] == 0 and counts["tc_pair_i16"] + counts["tc_pair_i16_ahead"] == 1, counts
    assert_same(dC.cpu().numpy(), expected(A, B, C, threads=16), f"{m}x{n}x{k}")


def test_small_problem_rule(gm):
    # beyond 256 rows, or above the work limit, the tensor-core path runs
    for (m, n, k) in ((257, 64, 64), (256, 1024, 2048)):
        A, B, C = gi.random_problem(840 + m + n, m, n, k, "i16")
        dA, dB, dC = (torch.from_numpy(x).cuda() for x in (A, B, C))
        counts = _kernel_counts(gm, lambda: gm.gemm_i16(dA, dB, dC))
        assert counts["skinny"] == 0 and counts["tc_pair_i16"] + counts["tc_pair_i16_ahead"] + counts["fused_i16"] == 1, counts
        assert_same(dC.cpu().numpy(), expected(A, B, C), f"{m}x{n}x{k}")
    # with the limit at 0 a small problem takes the tensor-core path too
    old = gm.get_option(gm.OPT_SMALL_MAX_MACS)
    gm.set_option(gm.OPT_SMALL_MAX_MACS, 0)
    try:
        A, B, C = gi.random_problem(850, 100, 300, 200, "i16")
        dA, dB, dC = (torch.from_numpy(x).cuda() for x in (A, B, C))
        counts = _kernel_counts(gm, lambda: gm.gemm_i16(dA, dB, dC))
        assert counts["skinny"] == 0 and counts["tc_pair_i16"] + counts["tc_pair_i16_ahead"] == 1, counts
        assert_same(dC.cpu().numpy(), expected(A, B, C), "limit 0")
    finally:
        gm.set_option(gm.OPT_SMALL_MAX_MACS, old)


def test_skinny_extremes(gm):
    for a, b in ((-32768, -32768), (-1, -1), (32767, -32768), (255, 255)):
        A = np.full((8, 2000), a, np.int16)
        B = np.full((2000, 300), b, np.int16)
        C = np.zeros((8, 300), np.int64)
        assert_same(run_gpu(gm, A, B, C), expected(A, B, C), f"skinny constant {(a, b)}")


@pytest.mark.parametrize("m", [8, 16])
def test_skinny_full_chunks_at_the_fp32_limit(gm, m):
    """One CTA per column block (ksplit 1), so every drain covers a full run of 256 reduction
    indices.  -32513 = 256 * (-128) + 255 makes both cross-term products -128 * 255 on every index:
    the cross sums reach -256 * 65280 = -16,711,680, within 2^24 = 16,777,216; 255 * 255 products
    drive the low sums, -32768 the high ones."""
    gm.set_option(gm.OPT_SKINNY_KSPLIT, 1)
    try:
        for a, b in ((-32513, -32513), (255, 255), (-32768, -32768), (-32513, 255), (32767, -32513)):
            A = np.full((m, 1024), a, np.int16)
            B = np.full((1024, 600), b, np.int16)
            C = gi.uniform_int(17, (m, 600), -(1 << 40), 1 << 40, np.int64)
            assert_same(run_gpu(gm, A, B, C), expected(A, B, C), f"skinny full chunks {(a, b)} m={m}")
    finally:
        gm.set_option(gm.OPT_SKINNY_KSPLIT, 0)


# ------------------------------------------------------------------ the five workloads
# The five workloads of the exact-GEMM problem statement (paper Section 4.1) are compared with the
# oracle on EVERY output element, at full size, on all host cores.  The int4 workload (a lower-
# precision extension, Section 6.1) is compared on sampled rows only; every one of its outputs is
# still covered by the row and column sums below.
FULL_WORKLOADS = ("i16_256", "i8_4096", "conv3x3_im2col", "i16_8192", "skinny_8x4096x4096")


def _sample_rows(m, count=24):
    rows = {0, 1, m - 1, m // 2, 127, 128, m - 129}
    rng = gi.uniform_int(4242 + m, (count,), 0, m - 1, np.int64)
    rows.update(int(r) for r in rng)
    return sorted(r for r in rows if 0 <= r < m)


def _check_sums(name, kind, A, B, C, got):
    """Every output through row and column sums (exact int64 arithmetic modulo 2^64): an extra
    check beside the element-wise comparison."""
    with np.errstate(over="ignore"):
        Bsum = B.astype(np.int64).sum(axis=1)
        row_exp = A.astype(np.int64) @ Bsum + C.astype(np.int64).sum(axis=1)
        Asum = A.astype(np.int64).sum(axis=0)
        col_exp = Asum @ B.astype(np.int64) + C.astype(np.int64).sum(axis=0)
        row_got = got.astype(np.int64).sum(axis=1)
        col_got = got.astype(np.int64).sum(axis=0)
    if kind != "i16":  # int32 C: the sums compare modulo 2^32
        row_exp, row_got, col_exp, col_got = (x & 0xFFFFFFFF for x in (row_exp, row_got, col_exp, col_got))
    assert np.array_equal(row_got, row_exp), f"{name}: row sums differ"
    assert np.array_equal(col_got, col_exp), f"{name}: column sums differ"


def test_five_workloads_are_listed():
    assert set(FULL_WORKLOADS) <= set(gi.WORKLOADS)


@pytest.mark.parametrize("name", FULL_WORKLOADS)
def test_workload_every_element(gm, name):
    """Full-size workload, every element of C against the oracle (all host cores)."""
    w = gi.WORKLOADS[name]
    A, B, C = gi.make_inputs(w)
    got = run_gpu(gm, A, B, C, w.kind)
    assert_same(got, expected(A, B, C, threads=oracle.host_cores()), f"{name} (all {w.m}x{w.n} outputs)")
    _check_sums(name, w.kind, A, B, C, got)


@pytest.mark.parametrize("name", [n for n in gi.WORKLOADS if n not in FULL_WORKLOADS])
def test_workload_sampled(gm, name):
    """Workloads beyond the five (int4 8192^3): sampled rows through the oracle, all outputs
    through row and column sums."""
    w = gi.WORKLOADS[name]
    A, B, C = gi.make_inputs(w)
    got = run_gpu(gm, A, B, C, w.kind)
    rows = _sample_rows(w.m)
    if w.kind == "i4":
        exp = C[rows].copy()
        oracle.gemm_i4(gi.pack_nibbles(A[rows]), gi.pack_nibbles(B), exp, w.k, nthreads=oracle.host_cores())
    else:
        exp = expected(A[rows], B, C[rows], threads=oracle.host_cores())
    assert_same(got[rows], exp, f"{name} sampled rows {rows[:4]}...")
    _check_sums(name, w.kind, A, B, C, got)


def test_read_probe_runs_clean(gm):
    """The skinny kernel's read floor probe (gemmi_stream_read_probe) streams a full-size B and a
    ragged one without a device-side failure."""
    for k, n in ((4096, 4096), (1000, 1000)):
        B = torch.zeros((k, n), dtype=torch.int16, device="cuda")
        gm.stream_read_probe(B)
        torch.cuda.synchronize()
        assert gm.device_status() == gm.OK


# ------------------------------------------------------------------ host-buffer API, streams, failure detection
def test_host_api_i16_and_i8(gm):
    A, B, C = gi.random_problem(900, 150, 170, 400, "i16")
    X = C.copy()
    gm.gemm_i16_host(A, B, X)
    assert_same(X, expected(A, B, C), "host i16")
    A, B, C = gi.random_problem(901, 150, 170, 400, "i8")
    X = C.copy()
    gm.gemm_i8_host(A, B, X)
    assert_same(X, expected(A, B, C), "host i8")


def test_host_api_padded(gm):
    m, n, k = 9, 50, 70
    A, B, C = gi.random_problem(902, m, n, k, "i16")
    big = np.full((m, n + 3), 7, np.int64)
    big[:, :n] = C
    gm.gemm_i16_host(A, B, big[:, :n])
    assert_same(big[:, :n], expected(A, B, C), "host padded")
    assert (big[:, n:] == 7).all()


# m >= 1024: the host path pipelines row panels of A and C (a ring of three device slots, so
# panels reuse slots) with B copied and split once.  From m = 1280 on, the first two and the last
# two panels are a quarter and a half panel (m = 2000: 128, 256, 208, 512, 512, 256, 128 rows;
# m = 8192: 128, 256, 256, fourteen of 512, 256, 128); m = 1024 and m = 1279 (512, 512, 255) keep
# whole panels.
@pytest.mark.parametrize("kind,m,n,k", [("i16", 2000, 300, 500), ("i8", 2000, 300, 500), ("i16", 1024, 64, 200),
                                        ("i16", 5000, 130, 96), ("i16", 8192, 72, 64), ("i8", 1280, 40, 80),
                                        ("i16", 1279, 24, 40)])
def test_host_api_pipelined_panels(gm, kind, m, n, k):
    A, B, C = gi.random_problem(905 + m + n, m, n, k, kind)
    # host operands with padded rows: the panel copies must honour the leading dimensions
    Ap = np.full((m, k + 5), 3, A.dtype)
    Ap[:, :k] = A
    Bp = np.full((k, n + 2), -3, B.dtype)
    Bp[:, :n] = B
    Cp = np.full((m, n + 1), 11, C.dtype)
    Cp[:, :n] = C
    (gm.gemm_i16_host if kind == "i16" else gm.gemm_i8_host)(Ap[:, :k], Bp[:, :n], Cp[:, :n])
    assert_same(Cp[:, :n], expected(A, B, C), f"host pipelined {kind} {m}x{n}x{k}")
    assert (Cp[:, n:] == 11).all()
    # a second call accumulates on top of the first (the slots and the split B are reused)
    (gm.gemm_i16_host if kind == "i16" else gm.gemm_i8_host)(Ap[:, :k], Bp[:, :n], Cp[:, :n])
    exp2 = expected(A, B, expected(A, B, C))
    assert_same(Cp[:, :n], exp2, "second pipelined call")


def test_non_default_stream(gm):
    A, B, C = gi.random_problem(903, 300, 260, 500, "i16")
    s = torch.cuda.Stream()
    dA, dB, dC = (torch.from_numpy(x).cuda() for x in (A, B, C))
    torch.cuda.synchronize()
    with torch.cuda.stream(s):
        gm.gemm_i16(dA, dB, dC)
    s.synchronize()
    assert_same(dC.cpu().numpy(), expected(A, B, C), "side stream")


def test_repeated_calls_accumulate(gm):
    A, B, C = gi.random_problem(904, 200, 140, 300, "i16")
    dA, dB, dC = (torch.from_numpy(x).cuda() for x in (A, B, C))
    for _ in range(3):
        gm.gemm_i16(dA, dB, dC)
    torch.cuda.synchronize()
    exp = C.copy()
    for _ in range(3):
        oracle.gemm(A, B, exp)
    assert_same(dC.cpu().numpy(), exp, "3x accumulate")


@pytest.mark.parametrize("m", [1, 8, 16])
def test_skinny_back_to_back_dependencies(gm, m):
    """Skinny launches may start while the previous kernel in the stream drains (programmatic
    dependent launch); each still has to see everything earlier kernels wrote.  Calls accumulate
    into one C, and between calls a torch kernel rewrites A in place, with no host
    synchronisation anywhere."""
    n, k = 700, 2000
    A, B, C = gi.random_problem(905 + m, m, n, k, "i16", a_range=(-1000, 1000))
    dA, dB, dC = (torch.from_numpy(x).cuda() for x in (A, B, C))
    exp = C.copy()
    a_host = A.copy()
    for r in range(6):
        gm.gemm_i16(dA, dB, dC)
        oracle.gemm(a_host, B, exp)
        dA.add_(r + 1)  # a torch kernel writes the next call's input
        a_host = (a_host.astype(np.int32) + r + 1).astype(np.int16)
    torch.cuda.synchronize()
    assert gm.device_status() == gm.OK
    assert_same(dC.cpu().numpy(), exp, f"m={m}: back-to-back skinny calls")


def test_bounded_wait_reports_timeout(gm):
    """A pipeline wait that can never complete gives up, reports, and leaves the context usable."""
    assert gm.selftest_wait_timeout(2000) == gm.ETIMEOUT
    assert (gm.device_status_detail() & 0xFF) == gm.ETIMEOUT
    assert gm.device_status() == gm.OK  # cleared
    A, B, C = gi.random_problem(905, 130, 130, 130, "i16")
    assert_same(run_gpu(gm, A, B, C), expected(A, B, C), "after timeout self-test")


def test_dtype_and_shape_errors(gm):
    a = torch.zeros((4, 4), dtype=torch.int32, device="cuda")
    with pytest.raises(TypeError):
        gm.gemm_i16(a, a, torch.zeros((4, 4), dtype=torch.int64, device="cuda"))
    with pytest.raises(ValueError):
        gm.gemm_i16(torch.zeros((4, 5), dtype=torch.int16, device="cuda"),
                    torch.zeros((4, 4), dtype=torch.int16, device="cuda"),
                    torch.zeros((4, 4), dtype=torch.int64, device="cuda"))


# ------------------------------------------------------------------ tuning options never change results
@pytest.mark.parametrize("opts", [
    {"OPT_TC_CHUNK_SCALE": 2}, {"OPT_TC_GROUP_M": 1}, {"OPT_TC_GROUP_M": 3, "OPT_TC_L2_HINTS": 1 | (2 << 2)},
    {"OPT_TC_CHUNK_SCALE": 2, "OPT_TC_L2_HINTS": 2 | (1 << 2)},
])
def test_tc_options_keep_results(gm, opts):
    saved = {k: gm.get_option(getattr(gm, k)) for k in opts}
    try:
        for k, v in opts.items():
            gm.set_option(getattr(gm, k), v)
        for kind, shape in (("i16", (300, 520, 1100)), ("i16", (129, 130, 4097)), ("i8", (260, 200, 2300))):
            A, B, C = gi.random_problem(1000 + sum(shape), *shape, kind)
            assert_same(run_gpu(gm, A, B, C), expected(A, B, C), f"{opts} {kind} {shape}")
    finally:
        for k, v in saved.items():
            gm.set_option(getattr(gm, k), v)


def test_calls_captured_in_a_cuda_graph(gm):
    """Calls captured into a CUDA graph replay exactly, and uncaptured calls still work afterwards."""
    s = torch.cuda.Stream()
    for kind, shape in (("i16", (300, 260, 700)), ("i16", (8, 1000, 900)), ("i8", (200, 130, 600))):
        A, B, C = gi.random_problem(1100 + sum(shape), *shape, kind)
        dA, dB = torch.from_numpy(A).cuda(), torch.from_numpy(B).cuda()
        dC = torch.from_numpy(C).cuda()
        fn = gm.gemm_i16 if kind == "i16" else gm.gemm_i8
        with torch.cuda.stream(s):
            fn(dA, dB, torch.from_numpy(C).cuda())  # warm-up outside the capture (workspace growth)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            fn(dA, dB, dC)
        dC.copy_(torch.from_numpy(C).cuda())
        g.replay()
        g.replay()
        torch.cuda.synchronize()
        exp = expected(A, B, C)
        oracle.gemm(A, B, exp)
        assert_same(dC.cpu().numpy(), exp, f"graph x2 {kind} {shape}")
        assert_same(run_gpu(gm, A, B, C), expected(A, B, C), f"uncaptured after graph {kind} {shape}")
