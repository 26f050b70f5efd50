"""GPU parity of the Karatsuba option (GEMMI_OPT_KARATSUBA): int16 C += A*B from three limb
products HH, LL and SS = (h_a + l_a)(h_b + l_b), bit for bit against the CPU oracle.

The limb sums s = h + l reach |s| = 255, so SS products reach 255^2 = 65025 and an SS chunk
(128 * CS reduction indices) reaches 128 * CS * 65025: within 2^23 at chunk scale 1 and within 2^24
(16,646,400 of 16,777,216) at chunk scale 2.  The constant operands below drive every product to
those limits; the shapes cross the SS, HH and LL chunk ends and ragged tiles.
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
    old = {o: gm.get_option(o) for o in (gm.OPT_KARATSUBA, gm.OPT_SMALL_MAX_MACS, gm.OPT_TC_CHUNK_SCALE)}
    gm.set_option(gm.OPT_KARATSUBA, 1)
    gm.set_option(gm.OPT_SMALL_MAX_MACS, 0)  # keep small problems on the tensor-core path
    yield gm
    for o, v in old.items():
        gm.set_option(o, v)


@pytest.fixture(params=[1, 2], ids=["chunks_2^23", "chunks_2^24"])
def chunk_scale(request, gm):
    gm.set_option(gm.OPT_TC_CHUNK_SCALE, request.param)
    yield request.param
    gm.set_option(gm.OPT_TC_CHUNK_SCALE, 2)


def expected(A, B, C):
    X = C.copy()
    oracle.gemm(A, B, X, nthreads=oracle.host_cores())
    return X


def run(gm, A, B, C):
    dA, dB, dC = (torch.from_numpy(np.ascontiguousarray(x)).cuda() for x in (A, B, C))
    gm.kernel_timing(True)
    gm.gemm_i16(dA, dB, dC)
    torch.cuda.synchronize()
    launches = gm.kernel_time(gm.KERNEL_TC_KARATSUBA)[1]
    gm.kernel_timing(False)
    assert gm.device_status() == gm.OK
    assert launches == 1, "the three-product kernel did not run"
    return dC.cpu().numpy()


def assert_same(got, exp, what):
    if not np.array_equal(got, exp):
        bad = np.argwhere(got != exp)
        i, j = bad[0]
        raise AssertionError(f"{what}: {len(bad)} mismatches, first at ({i},{j}): got {got[i, j]} want {exp[i, j]}")


@pytest.mark.parametrize("shape", [(17, 65, 1), (129, 127, 65), (300, 200, 290), (256, 384, 513), (200, 130, 1000),
                                   (130, 260, 2049), (512, 384, 290)])
def test_karatsuba_shapes(gm, shape, chunk_scale):
    m, n, k = shape
    A, B, C = gi.random_problem(700 + sum(shape), m, n, k, "i16")
    assert_same(run(gm, A, B, C), expected(A, B, C), f"Karatsuba {shape}")


@pytest.mark.parametrize("k", [127, 128, 129, 255, 256, 257, 511, 512, 513, 1023, 1024, 1025])
def test_karatsuba_chunk_boundaries(gm, k, chunk_scale):
    A, B, C = gi.random_problem(800 + k, 160, 136, k, "i16")
    assert_same(run(gm, A, B, C), expected(A, B, C), f"k={k}")


# 32639 = 256*127 + 127: limbs (127, 127), s = 254.  -32640 = 256*(-127) - 128: limbs (-127, -128),
# s = -255, the largest |s|.  32640: limbs (128, -128), s = 0, HH = LL = 2^14 in magnitude.
KA_EXTREMES = [(32639, 32639), (-32640, -32640), (32639, -32640), (-32768, -32768), (32767, 32767),
               (32640, 32640), (32767, -32768), (-1, -1)]


@pytest.mark.parametrize("ab", KA_EXTREMES)
def test_karatsuba_constant_extremes(gm, ab, chunk_scale):
    a, b = ab
    m, n, k = 200, 136, 2600
    A = np.full((m, k), a, np.int16)
    B = np.full((k, n), b, np.int16)
    C = gi.uniform_int(9, (m, n), -(1 << 40), 1 << 40, np.int64)
    assert_same(run(gm, A, B, C), expected(A, B, C), f"constant {ab} chunk scale {chunk_scale}")


def test_karatsuba_extreme_mixture(gm, chunk_scale):
    """Operands drawn from the extreme values only: sums that swing near the chunk bound with the low
    bits changing at every index."""
    vals = np.array([32639, -32640, 32640, -32768, 32767, -32641, 32641, -129], np.int16)
    m, n, k = 256, 256, 3000
    A = vals[gi.uniform_int(31, (m, k), 0, len(vals) - 1, np.int64)]
    B = vals[gi.uniform_int(32, (k, n), 0, len(vals) - 1, np.int64)]
    C = np.zeros((m, n), np.int64)
    assert_same(run(gm, A, B, C), expected(A, B, C), "extreme mixture")


def test_karatsuba_wraparound_mod_2_64(gm):
    A = np.full((130, 1024), -32768, np.int16)
    B = np.full((1024, 140), -32768, np.int16)
    C = np.full((130, 140), np.iinfo(np.int64).max - (1 << 35), np.int64)
    assert_same(run(gm, A, B, C), expected(A, B, C), "wrap-around")


def test_karatsuba_2048_cubed(gm):
    A, B, C = gi.random_problem(901, 2048, 2048, 2048, "i16")
    assert_same(run(gm, A, B, C), expected(A, B, C), "2048^3")
