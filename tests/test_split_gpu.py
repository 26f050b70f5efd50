"""GPU parity of the operand split on its two paths, through full GEMM calls against the oracle.

Operands whose base and row stride are 16-byte multiples are split by the TMA-fed kernel (raw
tiles through a shared-memory ring, B transposed through a swizzled staging tile and written
by TMA stores); others by the plain-load kernel.  The cases below put both paths through ragged
row counts (not a multiple of the 32-row A tile), reduction lengths that end inside a 64- or
128-element tile, column counts that end inside the 64/128-column B tile, padded leading
dimensions whose padding holds values that must not leak, and the packed-weight entry point.
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
    gm.set_option(gm.OPT_SKINNY_MAX_M, 0)
    gm.set_option(gm.OPT_FUSED_MAX_N, 0)
    yield gm
    gm.set_option(gm.OPT_SKINNY_MAX_M, 16)
    gm.set_option(gm.OPT_FUSED_MAX_N, 64)


def expected(A, B, C):
    X = C.copy()
    oracle.gemm(A, B, X, nthreads=8)
    return X


def padded(x, cols, fill):
    out = np.full((x.shape[0], cols), fill, x.dtype)
    out[:, :x.shape[1]] = x
    return torch.from_numpy(out).cuda()


def run(gm, A, B, C, lda, ldb):
    kind = "i16" if A.dtype == np.int16 else "i8"
    m, k = A.shape
    n = B.shape[1]
    big = 32000 if kind == "i16" else 120
    dA = padded(A, lda, big)[:, :k]
    dB = padded(B, ldb, -big)[:, :n]
    dC = torch.from_numpy(C.copy()).cuda()
    (gm.gemm_i16 if kind == "i16" else gm.gemm_i8)(dA, dB, dC)
    torch.cuda.synchronize()
    assert gm.device_status() == gm.OK
    return dC.cpu().numpy()


def assert_same(got, exp, what=""):
    if not np.array_equal(got, exp):
        bad = np.argwhere(got != exp)
        i, j = bad[0]
        raise AssertionError(f"{what}: {len(bad)} mismatches, first at ({i},{j}): got {got[i, j]} want {exp[i, j]}")


# (m, n, k, lda, ldb): TMA path (16-byte strides) then the plain-load path (odd strides)
CASES_I16 = [(77, 100, 200, 208, 104), (33, 64, 128, 128, 64), (1000, 600, 1000, 1000, 616), (250, 130, 72, 80, 136),
             (64, 200, 1000, 1003, 201), (31, 9, 17, 17, 9)]
CASES_I8 = [(77, 96, 208, 208, 112), (33, 128, 256, 256, 128), (700, 500, 1040, 1056, 512), (250, 144, 80, 96, 144),
            (64, 200, 1000, 1001, 203), (31, 9, 17, 17, 9)]


@pytest.mark.parametrize("case", CASES_I16)
def test_split_i16_layouts(gm, case):
    m, n, k, lda, ldb = case
    A, B, C = gi.random_problem(6100 + sum(case), m, n, k, "i16")
    assert_same(run(gm, A, B, C, lda, ldb), expected(A, B, C), f"i16 {case}")


@pytest.mark.parametrize("case", CASES_I8)
def test_split_i8_layouts(gm, case):
    m, n, k, lda, ldb = case
    A, B, C = gi.random_problem(6200 + sum(case), m, n, k, "i8")
    assert_same(run(gm, A, B, C, lda, ldb), expected(A, B, C), f"i8 {case}")


@pytest.mark.parametrize("kind", ["i16", "i8"])
def test_split_packed_weights_padded(gm, kind):
    m, n, k = 300, 200, 400
    A, B, C = gi.random_problem(6300, m, n, k, kind)
    ldb = n + (8 if kind == "i16" else 16)
    dB = padded(B, ldb, 7)[:, :n]
    packed = (gm.pack_b_i16 if kind == "i16" else gm.pack_b_i8)(dB)
    try:
        dA, dC = torch.from_numpy(A).cuda(), torch.from_numpy(C.copy()).cuda()
        (gm.gemm_i16_packed if kind == "i16" else gm.gemm_i8_packed)(dA, packed, dC)
        torch.cuda.synchronize()
        assert gm.device_status() == gm.OK
        assert_same(dC.cpu().numpy(), expected(A, B, C), f"packed {kind}")
    finally:
        packed.close()
