"""Parity at sizes beyond the benchmark workloads: int16 16384^3, a 2^20-row narrow-output GEMM
(the convolution shape at ten times the batch) and int4 16384^3.

The narrow-output GEMM (3.9e10 multiply-adds) is compared with the oracle on every element.  The
two 16384^3 cases are SAMPLED: the oracle computes sampled rows (4.4e12 multiply-adds for all of
them would take minutes on the host), and every other entry is checked through its row and column
sums, computed in exact integer arithmetic (numpy int64, which wraps modulo 2^64 like the
library's int64 C; int32 results compare modulo 2^32).  Inputs are drawn in row blocks from the
same counter-based generator as every other test, so host memory stays a few GB.
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


def draw(seed, rows, cols, lo, hi, dtype, block=2048):
    out = np.empty((rows, cols), dtype)
    for r0 in range(0, rows, block):
        r1 = min(rows, r0 + block)
        out[r0:r1] = gi._draw_rows(seed, rows, cols, r0, r1 - r0, ("uniform", lo, hi), dtype)
    return out


def sample_rows(m, count=12, seed=0):
    rows = {0, 1, m - 1, m // 2, 127, 128, 129}
    rows.update(int(r) for r in gi.uniform_int(seed, (count,), 0, m - 1, np.int64))
    return sorted(r for r in rows if 0 <= r < m)


def check_sums(got, A, B, C, bits, block=2048):
    """Row and column sums of C + A @ B (C None: zero) against those of the device result, modulo
    2^bits (row blocks at a time, so no full-size int64 copy of A or B is made)."""
    m, k = A.shape
    n = B.shape[1]
    with np.errstate(over="ignore"):
        bsum = B.sum(axis=1, dtype=np.int64)
        asum = A.sum(axis=0, dtype=np.int64)
        row_exp = C.sum(axis=1, dtype=np.int64) if C is not None else np.zeros(m, np.int64)
        for r0 in range(0, m, block):
            row_exp[r0:r0 + block] += A[r0:r0 + block].astype(np.int64) @ bsum
        col_exp = C.sum(axis=0, dtype=np.int64) if C is not None else np.zeros(n, np.int64)
        for p0 in range(0, k, block):
            col_exp += asum[p0:p0 + block] @ B[p0:p0 + block].astype(np.int64)
        row_got = got.sum(axis=1, dtype=np.int64)
        col_got = got.sum(axis=0, dtype=np.int64)
    for name, e, g in (("row", row_exp, row_got), ("column", col_exp, col_got)):
        if bits < 64:
            e, g = e & ((1 << bits) - 1), g & ((1 << bits) - 1)
        assert np.array_equal(e, g), f"{name} sums differ at {np.argwhere(e != g)[:3].ravel().tolist()}"


def test_int16_16384_cubed_sampled(gm):
    n = 16384
    A = draw(40001, n, n, -32768, 32767, np.int16)
    B = draw(40002, n, n, -32768, 32767, np.int16)
    dA, dB = torch.from_numpy(A).cuda(), torch.from_numpy(B).cuda()
    dC = torch.zeros((n, n), dtype=torch.int64, device="cuda")
    gm.gemm_i16(dA, dB, dC)
    torch.cuda.synchronize()
    assert gm.device_status() == gm.OK
    got = dC.cpu().numpy()
    del dA, dB, dC
    rows = sample_rows(n, seed=40003)
    exp = np.zeros((len(rows), n), np.int64)
    oracle.gemm(A[rows], B, exp, nthreads=oracle.host_cores())
    assert np.array_equal(got[rows], exp)
    check_sums(got, A, B, None, 64)


def test_narrow_output_2_pow_20_rows_every_element(gm):
    m, n, k = 1 << 20, 64, 576
    A = draw(40011, m, k, -32768, 32767, np.int16)
    B = draw(40012, k, n, -32768, 32767, np.int16)
    C = draw(40013, m, n, -(1 << 40), 1 << 40, np.int64)
    dA, dB, dC = (torch.from_numpy(x).cuda() for x in (A, B, C))
    gm.gemm_i16(dA, dB, dC)
    torch.cuda.synchronize()
    assert gm.device_status() == gm.OK
    got = dC.cpu().numpy()
    del dA, dB, dC
    exp = C.copy()
    oracle.gemm(A, B, exp, nthreads=oracle.host_cores())
    assert np.array_equal(got, exp)
    check_sums(got, A, B, C, 64)


def test_int4_16384_cubed_sampled(gm):
    n = 16384
    A = draw(40021, n, n, -8, 7, np.int8)
    B = draw(40022, n, n, -8, 7, np.int8)
    Ap, Bp = gi.pack_nibbles(A), gi.pack_nibbles(B)
    dC = torch.zeros((n, n), dtype=torch.int32, device="cuda")
    gm.gemm_i4(torch.from_numpy(Ap).cuda(), torch.from_numpy(Bp).cuda(), dC, n)
    torch.cuda.synchronize()
    assert gm.device_status() == gm.OK
    got = dC.cpu().numpy()
    del dC
    rows = sample_rows(n, seed=40023)
    exp = np.zeros((len(rows), n), np.int32)
    oracle.gemm_i4(Ap[rows], Bp, exp, n, nthreads=oracle.host_cores())
    assert np.array_equal(got[rows], exp)
    check_sums(got, A, B, None, 32)
