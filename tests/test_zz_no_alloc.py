"""gemm_i16_noalloc: the int16 GEMM for callers that cannot allocate device memory at call time.

Such callers (an inference server that gave all free device memory to its own pool, a loop
that cannot absorb the synchronisation of growing a buffer) get an entry point whose scratch
is a fixed array inside the library instead of a workspace it allocates.  This file checks,
through the C ABI, that it returns exactly what gemm_i16 returns, on two calls in a row that
share that array, and that a problem too large for the array is refused.  It sits last in
collection order so that a run stopping at the first failure has already run everything else.
"""
import ctypes

import numpy as np
import pytest

import gemm_inputs as gi

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
    return lib


def _call_noalloc(L, dA, dB, dC):
    m, k = dA.shape
    n = dB.shape[1]
    stream = torch.cuda.current_stream().cuda_stream
    return L.gemm_i16_noalloc(m, n, k, dA.data_ptr(), dA.stride(0), dB.data_ptr(), dB.stride(0),
                              dC.data_ptr(), dC.stride(0), stream)


def test_noalloc_matches_gemm_i16_on_two_calls(L):
    import paper_2302_07594_gb300 as gm
    # two different problems back to back: the second reuses the scratch the first left behind
    for seed, (m, n, k) in ((11, (300, 200, 700)), (12, (1000, 1100, 2500))):
        A, B, C = gi.random_problem(seed, m, n, k, "i16")
        dA, dB = torch.from_numpy(A).cuda(), torch.from_numpy(B).cuda()
        want = torch.from_numpy(C).cuda()
        got = torch.from_numpy(C).cuda()
        gm.gemm_i16(dA, dB, want)                      # the existing entry point
        assert _call_noalloc(L, dA, dB, got) == gm.OK, gm.last_error()
        torch.cuda.synchronize()
        assert gm.device_status() == gm.OK
        w, g = want.cpu().numpy(), got.cpu().numpy()
        assert np.array_equal(g, w), f"noalloc differs from gemm_i16 for {(m, n, k)}"


def test_noalloc_rejects_problems_beyond_its_scratch(L):
    import paper_2302_07594_gb300 as gm
    m = n = k = 4096  # 4*(m+n)*k bytes of limb planes = 128 MiB > 32 MiB
    dA = torch.zeros((m, k), dtype=torch.int16, device="cuda")
    dB = torch.zeros((k, n), dtype=torch.int16, device="cuda")
    dC = torch.zeros((m, n), dtype=torch.int64, device="cuda")
    assert _call_noalloc(L, dA, dB, dC) == gm.EINVAL
    assert "scratch" in gm.last_error()
