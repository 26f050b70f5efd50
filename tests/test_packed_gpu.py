"""Pre-packed weights (Section 5.1 of the paper): pack B once, run many A through it.

Results must equal the CPU oracle bit for bit, exactly as gemm_i16 / gemm_i8 do.
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
    assert torch.cuda.is_available()
    gm.lib()
    return gm


def _oracle(A, B, C):
    X = C.copy()
    oracle.gemm(A, B, X, nthreads=8)
    return X


@pytest.mark.parametrize("kind", ["i16", "i8"])
@pytest.mark.parametrize("kn", [(576, 64), (290, 300), (1, 7), (1025, 129)])
def test_packed_matches_oracle_for_several_A(gm, kind, kn):
    k, n = kn
    _, B, _ = gi.random_problem(1200 + k + n, 1, n, k, kind)
    dB = torch.from_numpy(B).cuda()
    pack = gm.pack_b_i16 if kind == "i16" else gm.pack_b_i8
    run = gm.gemm_i16_packed if kind == "i16" else gm.gemm_i8_packed
    Bp = pack(dB)
    del dB  # the packed copy is independent of the original buffer
    torch.cuda.synchronize()
    for idx, m in enumerate((3, 130, 257)):
        A, _, C = gi.random_problem(1300 + idx + k, m, n, k, kind)
        dA, dC = torch.from_numpy(A).cuda(), torch.from_numpy(C).cuda()
        run(dA, Bp, dC)
        torch.cuda.synchronize()
        assert np.array_equal(dC.cpu().numpy(), _oracle(A, B, C)), f"{kind} m={m} k={k} n={n}"
    Bp.close()
    with pytest.raises(ValueError):
        run(dA, Bp, dC)


def test_packed_conv_workload_every_element(gm):
    """The im2col workload with its weights packed once: every element against the oracle."""
    w = gi.WORKLOADS["conv3x3_im2col"]
    A, B, C = gi.make_inputs(w)
    Bp = gm.pack_b_i16(torch.from_numpy(B).cuda())
    dA, dC = torch.from_numpy(A).cuda(), torch.from_numpy(C).cuda()
    gm.gemm_i16_packed(dA, Bp, dC)
    torch.cuda.synchronize()
    got = dC.cpu().numpy()
    exp = C.copy()
    oracle.gemm(A, B, exp, nthreads=oracle.host_cores())
    assert np.array_equal(got, exp)


def test_packed_rejects_mismatches(gm):
    Bp = gm.pack_b_i16(torch.zeros((64, 32), dtype=torch.int16, device="cuda"))
    with pytest.raises(ValueError):
        gm.gemm_i16_packed(torch.zeros((8, 63), dtype=torch.int16, device="cuda"), Bp,
                           torch.zeros((8, 32), dtype=torch.int64, device="cuda"))
    with pytest.raises(TypeError):
        gm.gemm_i8_packed(torch.zeros((8, 64), dtype=torch.int8, device="cuda"), Bp,
                          torch.zeros((8, 32), dtype=torch.int32, device="cuda"))
    Bp.close()
