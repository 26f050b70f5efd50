"""gemm_i16_noalloc: the int16 GEMM for callers that cannot allocate device memory at call time.

Such callers (an inference server that gave all free device memory to its own pool, a loop
that cannot absorb the synchronisation of growing a buffer) get an entry point whose scratch
is a fixed array inside the library instead of a workspace it allocates.  This file checks,
through the C ABI, that it returns exactly what the oracle and gemm_i16 return, on two calls in
a row that share that array and on a problem at the array's size limit; that a problem too
large for the array is refused; and that a pipeline wait that runs out inside this entry
point's status word is reported by the status calls.  It sits last in collection order so that
a run stopping at the first failure has already run everything else.
"""
import ctypes

import numpy as np
import pytest

import gemm_inputs as gi
import oracle

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def L():
    import paper_2302_07594_gb300 as gm
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    lib = gm.lib()
    f = lib.gemm_i16_noalloc
    f.argtypes = [ctypes.c_int64] * 3 + [ctypes.c_void_p, ctypes.c_int64] * 3 + [ctypes.c_void_p]
    f.restype = ctypes.c_int
    lib.gemmi_device_status_stream.argtypes = [ctypes.c_void_p]
    lib.gemmi_device_status_stream.restype = ctypes.c_int
    lib.gemmi_noalloc_selftest_wait_timeout.argtypes = [ctypes.c_int64, ctypes.c_void_p]
    lib.gemmi_noalloc_selftest_wait_timeout.restype = ctypes.c_int
    return lib


def _stream():
    return torch.cuda.current_stream().cuda_stream


def _call_noalloc(L, dA, dB, dC):
    m, k = dA.shape
    n = dB.shape[1]
    return L.gemm_i16_noalloc(m, n, k, dA.data_ptr(), dA.stride(0), dB.data_ptr(), dB.stride(0),
                              dC.data_ptr(), dC.stride(0), _stream())


def _oracle(A, B, C):
    X = C.copy()
    oracle.gemm(A, B, X, nthreads=oracle.host_cores())
    return X


def _check_problem(L, seed, m, n, k):
    import paper_2302_07594_gb300 as gm
    A, B, C = gi.random_problem(seed, m, n, k, "i16")
    dA, dB = torch.from_numpy(A).cuda(), torch.from_numpy(B).cuda()
    want = torch.from_numpy(C).cuda()
    got = torch.from_numpy(C).cuda()
    gm.gemm_i16(dA, dB, want)                      # the existing entry point
    assert _call_noalloc(L, dA, dB, got) == gm.OK, gm.last_error()
    assert L.gemmi_device_status_stream(_stream()) == gm.OK, gm.last_error()
    g = got.cpu().numpy()
    assert np.array_equal(g, _oracle(A, B, C)), f"noalloc differs from the oracle for {(m, n, k)}"
    assert np.array_equal(g, want.cpu().numpy()), f"noalloc differs from gemm_i16 for {(m, n, k)}"


def test_noalloc_matches_oracle_and_gemm_i16_on_two_calls(L):
    # two different problems back to back: the second reuses the scratch the first left behind
    for seed, (m, n, k) in ((11, (300, 200, 700)), (12, (1000, 1100, 2500))):
        _check_problem(L, seed, m, n, k)


def test_noalloc_at_the_scratch_limit(L):
    import paper_2302_07594_gb300 as gm
    m = n = k = 2000  # 4*(m+n)*k + 256 = 32,000,256 bytes of the 33,554,432-byte array
    assert 4 * (m + n) * k + 256 <= gm.NOALLOC_SCRATCH_BYTES
    _check_problem(L, 13, m, n, k)


def test_noalloc_rejects_problems_beyond_its_scratch(L):
    import paper_2302_07594_gb300 as gm
    m = n = k = 4096  # 4*(m+n)*k bytes of limb planes = 128 MiB > 32 MiB
    dA = torch.zeros((m, k), dtype=torch.int16, device="cuda")
    dB = torch.zeros((k, n), dtype=torch.int16, device="cuda")
    dC = torch.zeros((m, n), dtype=torch.int64, device="cuda")
    assert _call_noalloc(L, dA, dB, dC) == gm.EINVAL
    assert "scratch" in gm.last_error()


def test_noalloc_status_word_reports_a_wait_that_ran_out(L):
    """A probe wait that nothing completes runs out in this entry point's status word; the status
    calls report it once and clear it, and the array still serves a correct GEMM afterwards."""
    import paper_2302_07594_gb300 as gm
    assert L.gemmi_noalloc_selftest_wait_timeout(2000, _stream()) == gm.OK, gm.last_error()
    assert L.gemmi_device_status_stream(_stream()) == gm.ETIMEOUT
    assert "ran out of time" in gm.last_error()
    assert gm.device_status() == gm.OK          # cleared by the read above
    assert L.gemmi_noalloc_selftest_wait_timeout(2000, _stream()) == gm.OK, gm.last_error()
    assert gm.device_status() == gm.ETIMEOUT     # the whole-device read sees it too
    assert L.gemmi_device_status_stream(_stream()) == gm.OK
    _check_problem(L, 14, 130, 140, 150)
