"""GPU parity of gemm_i16_srs: the paper's micro-kernel output, int16 C += srs(A*B, shift).

The exact product comes from the regular int16 paths (skinny for m <= 16, the
narrow-n fused kernel for n <= 64, the general tensor-core kernel otherwise);
a requantising pass then shifts with rounding half up, saturates to int16 and
adds modulo 2^16.  Expected values come from oracle.gemm_srs on the same seeded
inputs, bit for bit.
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


def expected(A, B, C, shift):
    X = C.copy()
    oracle.gemm_srs(A, B, X, shift, nthreads=8)
    return X


def run(gm, A, B, C, shift):
    dA, dB, dC = (torch.from_numpy(np.ascontiguousarray(x)).cuda() for x in (A, B, C))
    gm.gemm_i16_srs(dA, dB, dC, shift)
    torch.cuda.synchronize()
    assert gm.device_status() == gm.OK
    return dC.cpu().numpy()


def assert_same(got, exp, what=""):
    if not np.array_equal(got, exp):
        bad = np.argwhere(got != exp)
        i, j = bad[0]
        raise AssertionError(f"{what}: {len(bad)} mismatches, first at ({i},{j}): got {got[i, j]} want {exp[i, j]}")


# (m, n, k): skinny (m <= 16), fused narrow-n (n <= 64, k % 8 == 0), general tensor-core path
SHAPES = [(8, 300, 500), (16, 1000, 64), (200, 64, 576), (300, 40, 128), (260, 300, 700), (129, 130, 2049)]
SHIFTS = [0, 1, 7, 15, 20, 26, 31, 40]


@pytest.mark.parametrize("shape", SHAPES)
@pytest.mark.parametrize("shift", SHIFTS)
def test_srs_shapes_and_shifts(gm, shape, shift):
    m, n, k = shape
    A, B, _ = gi.random_problem(800 + sum(shape), m, n, k, "i16")
    C = gi.uniform_int(801 + m, (m, n), -32768, 32767, np.int16)
    assert_same(run(gm, A, B, C, shift), expected(A, B, C, shift), f"{shape} shift {shift}")


@pytest.mark.parametrize("shift", [0, 9, 22])
def test_srs_small_values_no_saturation(gm, shift):
    # sums inside int16 at shift 0: the rounding and the wrap carry the result
    A, B, _ = gi.random_problem(810, 150, 170, 300, "i16", a_range=(-9, 9), b_range=(-9, 9))
    C = gi.uniform_int(811, (150, 170), -32768, 32767, np.int16)
    assert_same(run(gm, A, B, C, shift), expected(A, B, C, shift), f"small values shift {shift}")


@pytest.mark.parametrize("ab", [(-32768, -32768), (32767, -32768), (32767, 32767), (1, 1), (-1, 1)])
def test_srs_constant_operands(gm, ab):
    a, b = ab
    for m in (4, 200):
        A = np.full((m, 1500), a, np.int16)
        B = np.full((1500, 72), b, np.int16)
        C = gi.uniform_int(812 + m, (m, 72), -32768, 32767, np.int16)
        for shift in (0, 11, 30, 34):
            assert_same(run(gm, A, B, C, shift), expected(A, B, C, shift), f"constant {ab} m={m} shift {shift}")


def test_srs_padded_and_misaligned_C(gm):
    m, n, k = 140, 77, 300
    A, B, _ = gi.random_problem(813, m, n, k, "i16")
    C = gi.uniform_int(814, (m, n), -32768, 32767, np.int16)
    exp = expected(A, B, C, 12)
    for ldc, off in ((81, 0), (84, 1), (80, 0)):
        buf = gi.uniform_int(815 + ldc, (m, ldc), -32768, 32767, np.int16)
        buf[:, off:off + n] = C
        dA, dB = torch.from_numpy(A).cuda(), torch.from_numpy(B).cuda()
        dbuf = torch.from_numpy(buf).cuda()
        gm.gemm_i16_srs(dA, dB, dbuf[:, off:off + n], 12)
        torch.cuda.synchronize()
        got = dbuf.cpu().numpy()
        assert_same(got[:, off:off + n], exp, f"ldc={ldc} offset={off}")
        outside = np.ones(buf.shape, bool)
        outside[:, off:off + n] = False
        assert np.array_equal(got[outside], buf[outside]), f"ldc={ldc}: entries outside C were written"


def test_srs_repeated_calls_and_empty(gm):
    A, B, _ = gi.random_problem(816, 100, 90, 200, "i16")
    C = gi.uniform_int(817, (100, 90), -32768, 32767, np.int16)
    dA, dB, dC = (torch.from_numpy(x).cuda() for x in (A, B, C))
    exp = C.copy()
    for shift in (3, 17, 25):
        gm.gemm_i16_srs(dA, dB, dC, shift)
        oracle.gemm_srs(A, B, exp, shift)
    torch.cuda.synchronize()
    assert_same(dC.cpu().numpy(), exp, "three calls in a row")
    # k == 0 leaves C unchanged
    Z = torch.zeros((100, 0), dtype=torch.int16, device="cuda")
    Zb = torch.zeros((0, 90), dtype=torch.int16, device="cuda")
    before = dC.clone()
    gm.gemm_i16_srs(Z, Zb, dC, 5)
    torch.cuda.synchronize()
    assert torch.equal(before, dC)
    with pytest.raises(gm.GemmiError):
        gm.gemm_i16_srs(dA, dB, dC, 63)
