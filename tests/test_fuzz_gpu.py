"""Randomized parity sweep: seeded shapes, paddings, operand types and dispatch options.

Each case draws m, n, k (edge values and ranges that cross tile, chunk and stage boundaries), padded
leading dimensions, an operand type (int16, int8, int4) and a setting of the dispatch options (SM
pairs on or off, the skinny and narrow-n paths on or off, the exact-chunk length), runs the GEMM on
the device and compares every entry with the oracle.  The draws come from one fixed seed, so the
sweep is the same on every run.
"""
import numpy as np
import pytest

import gemm_inputs as gi
import oracle

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

EDGE = [1, 2, 3, 7, 8, 15, 16, 17, 31, 33, 63, 64, 65, 127, 128, 129, 255, 256, 257]


def draw_cases(count=240, seed=20230215):
    rng = np.random.default_rng(seed)

    def dim(lo, hi):
        return int(rng.choice(EDGE)) if rng.random() < 0.4 else int(rng.integers(lo, hi + 1))

    cases = []
    for i in range(count):
        kind = ("i16", "i8", "i4")[i % 3]
        m, n, k = dim(1, 700), dim(1, 600), dim(1, 2200)
        pad = [int(rng.integers(0, 3)) * int(rng.choice([1, 7, 16])) for _ in range(3)]
        opts = {"OPT_TC_PAIR": int(rng.integers(0, 2)), "OPT_SKINNY_MAX_M": int(rng.choice([0, 16])),
                "OPT_FUSED_MAX_N": int(rng.choice([0, 64])), "OPT_TC_CHUNK_SCALE": int(rng.integers(1, 3))}
        cases.append((i, kind, m, n, k, pad, opts))
    return cases


@pytest.fixture(scope="module")
def gm():
    import paper_2302_07594_gb300 as gm
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    gm.lib()
    names = ("OPT_TC_PAIR", "OPT_SKINNY_MAX_M", "OPT_FUSED_MAX_N", "OPT_TC_CHUNK_SCALE")
    saved = {nm: gm.get_option(getattr(gm, nm)) for nm in names}
    yield gm
    for nm, v in saved.items():
        gm.set_option(getattr(gm, nm), v)


def padded_device(x, extra, fill):
    rows, cols = x.shape
    buf = np.full((rows, cols + extra), fill, x.dtype)
    buf[:, :cols] = x
    return torch.from_numpy(buf).cuda()[:, :cols]


@pytest.mark.parametrize("case", draw_cases(), ids=lambda c: f"{c[0]}-{c[1]}-{c[2]}x{c[3]}x{c[4]}")
def test_random_case_matches_oracle(gm, case):
    idx, kind, m, n, k, pad, opts = case
    for nm, v in opts.items():
        gm.set_option(getattr(gm, nm), v)
    A, B, C = gi.random_problem(30000 + idx, m, n, k, kind)
    exp = C.copy()
    if kind == "i4":
        Ap, Bp = gi.pack_nibbles(A), gi.pack_nibbles(B)
        oracle.gemm_i4(Ap, Bp, exp, k, nthreads=8)
        dA, dB = padded_device(Ap, pad[0], 0x5A), padded_device(Bp, pad[1], 0xA5)
        dC = padded_device(C, pad[2], 7)
        gm.gemm_i4(dA, dB, dC, k)
    else:
        oracle.gemm(A, B, exp, nthreads=8)
        big = 12345 if kind == "i16" else 99
        dA, dB = padded_device(A, pad[0], big), padded_device(B, pad[1], -big)
        dC = padded_device(C, pad[2], 7)
        (gm.gemm_i16 if kind == "i16" else gm.gemm_i8)(dA, dB, dC)
    torch.cuda.synchronize()
    assert gm.device_status() == gm.OK
    got = dC.cpu().numpy()
    if not np.array_equal(got, exp):
        bad = np.argwhere(got != exp)
        i, j = bad[0]
        raise AssertionError(f"case {case}: {len(bad)} mismatches, first at ({i},{j}): got {got[i, j]} want {exp[i, j]}")
