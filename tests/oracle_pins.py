"""Checks that pin the CPU oracle to facts fixed outside itself.

Each check returns a list of failure strings (empty = pass) so the same
checks serve both the regular tests and the mutation tests, which plant a
mistake in a copy of the oracle's C source and require some check to fail.

What pins the oracle (the GEMM definition of Section 4.1, C += A*B):
  * hand-computed cases (tests/golden/hand_cases.json), each with its working;
  * brute force with Python's arbitrary-precision integers on tiny shapes;
  * numpy's integer matmul on int64 arrays (an exact library routine);
  * closed forms: all-ones gives C += k, extreme operands give k*2^30 etc.;
  * identity and permutation matrices;
  * the paper's blocked algorithm (Figure 1, loops L1-L3): summing the GEMM
    over k_c-blocks of the reduction dimension and m_c/n_c-blocks of C gives
    the unblocked result;
  * modular wrap-around and untouched padding outside the m x n block of C.
"""
from __future__ import annotations

import json
import os

import numpy as np

import gemm_inputs as gi
import oracle

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "hand_cases.json")
TINY = (0, 1, 2, 3, 5, 8, 17)


def golden_cases():
    with open(GOLDEN) as f:
        return json.load(f)["cases"]


def _arrays(case):
    op = np.int16 if case["kind"] == "i16" else np.int8
    cd = np.int64 if case["kind"] == "i16" else np.int32
    A = np.array(case["A"], dtype=op).reshape(case["m"], case["k"])
    B = np.array(case["B"], dtype=op).reshape(case["k"], case["n"])
    C = np.array(case["C_in"], dtype=cd).reshape(case["m"], case["n"])
    E = np.array(case["C_out"], dtype=cd).reshape(case["m"], case["n"])
    return A, B, C, E


def bigint_gemm(A, B, C, bits):
    """C + A*B with Python integers, reduced to a two's-complement `bits`-bit value."""
    m, k = A.shape
    n = B.shape[1]
    out = np.empty_like(C)
    mod = 1 << bits
    for i in range(m):
        for j in range(n):
            s = int(C[i, j])
            for p in range(k):
                s += int(A[i, p]) * int(B[p, j])
            s %= mod
            if s >= mod >> 1:
                s -= mod
            out[i, j] = s
    return out


def numpy_gemm(A, B, C):
    """C + A*B through numpy's exact int64 matmul (wraps modulo 2^64)."""
    P = np.matmul(A.astype(np.int64), B.astype(np.int64))
    with np.errstate(over="ignore"):
        R = C.astype(np.int64) + P
    return R.astype(C.dtype)  # int32 C: astype keeps the low 32 bits (mod 2^32)


def _run(lib, A, B, C, nthreads=1):
    X = C.copy()
    oracle.gemm(A, B, X, nthreads=nthreads, lib=lib)
    return X


def check_golden(lib):
    bad = []
    for case in golden_cases():
        A, B, C, E = _arrays(case)
        got = _run(lib, A, B, C)
        if not np.array_equal(got, E):
            bad.append(f"golden {case['name']}: {got.tolist()} != {E.tolist()}")
    return bad


def check_bruteforce(lib, shapes=None, kinds=("i16", "i8")):
    bad = []
    shapes = shapes or [(m, n, k) for m in TINY for n in TINY for k in TINY]
    for kind in kinds:
        bits = 64 if kind == "i16" else 32
        for idx, (m, n, k) in enumerate(shapes):
            A, B, C = gi.random_problem(7000 + idx, m, n, k, kind)
            exp = bigint_gemm(A, B, C, bits)
            got = _run(lib, A, B, C)
            if not np.array_equal(got, exp):
                bad.append(f"bruteforce {kind} {m}x{n}x{k}")
    return bad


def check_extreme_bruteforce(lib):
    """All-minimum / all-maximum operands, where any int32 shortcut overflows."""
    bad = []
    for kind, lo, hi in (("i16", -32768, 32767), ("i8", -128, 127)):
        op = np.int16 if kind == "i16" else np.int8
        cd = np.int64 if kind == "i16" else np.int32
        bits = 64 if kind == "i16" else 32
        for (m, n, k) in ((3, 5, 17), (8, 2, 33), (1, 1, 130)):
            for a, b in ((lo, lo), (hi, lo), (hi, hi)):
                A = np.full((m, k), a, op)
                B = np.full((k, n), b, op)
                C = np.zeros((m, n), cd)
                if not np.array_equal(_run(lib, A, B, C), bigint_gemm(A, B, C, bits)):
                    bad.append(f"extreme {kind} {m}x{n}x{k} a={a} b={b}")
    return bad


def check_numpy(lib, shapes=((64, 48, 80), (129, 70, 301), (256, 256, 256))):
    bad = []
    for idx, (m, n, k) in enumerate(shapes):
        for kind in ("i16", "i8"):
            A, B, C = gi.random_problem(9100 + idx, m, n, k, kind)
            if not np.array_equal(_run(lib, A, B, C), numpy_gemm(A, B, C)):
                bad.append(f"numpy {kind} {m}x{n}x{k}")
    return bad


def check_closed_forms(lib):
    bad = []
    for k in (1, 2, 7, 300):
        m, n = 3, 4
        ones = _run(lib, np.ones((m, k), np.int16), np.ones((k, n), np.int16), np.zeros((m, n), np.int64))
        if not (ones == k).all():
            bad.append(f"all-ones k={k}")
        mm = _run(lib, np.full((m, k), -32768, np.int16), np.full((k, n), -32768, np.int16),
                  np.zeros((m, n), np.int64))
        if not (mm == k * (1 << 30)).all():
            bad.append(f"min*min k={k}")
        xm = _run(lib, np.full((m, k), 32767, np.int16), np.full((k, n), -32768, np.int16),
                  np.zeros((m, n), np.int64))
        if not (xm == -k * 1073709056).all():
            bad.append(f"max*min k={k}")
        i8 = _run(lib, np.full((m, k), -128, np.int8), np.full((k, n), -128, np.int8),
                  np.zeros((m, n), np.int32))
        if not (i8 == k * 16384).all():  # k * 2^14 < 2^31 for every k here
            bad.append(f"i8 min*min k={k}")
    return bad


def check_identity_permutation(lib):
    bad = []
    m, n = 37, 23
    _, B, C = gi.random_problem(31, m, n, m, "i16")
    eye = np.eye(m, dtype=np.int16)
    if not np.array_equal(_run(lib, eye, B, C), C + B.astype(np.int64)):
        bad.append("identity")
    perm = np.array(gi.uniform_int(77, (m,), 0, 1 << 30, np.int64).argsort(kind="stable"))
    P = np.zeros((m, m), np.int16)
    P[np.arange(m), perm] = 1
    if not np.array_equal(_run(lib, P, B, C), C + B[perm].astype(np.int64)):
        bad.append("permutation")
    return bad


def check_blocked(lib, m=70, n=45, k=133, mc=32, nc=16, kc=40):
    """Figure 1 of the paper: loops L1 (n_c), L2 (k_c), L3 (m_c) around C += A_c B_c."""
    A, B, C = gi.random_problem(55, m, n, k, "i16")
    full = _run(lib, A, B, C)
    X = C.copy()
    for jc in range(0, n, nc):
        for pc in range(0, k, kc):
            for ic in range(0, m, mc):
                sub = X[ic:ic + mc, jc:jc + nc]  # a strided view: leading dimension n
                oracle.gemm(A[ic:ic + mc, pc:pc + kc], B[pc:pc + kc, jc:jc + nc], sub, lib=lib)
    return [] if np.array_equal(full, X) else ["blocked"]


def check_padding(lib):
    """Leading dimensions larger than the rows: only the m x n block of C changes."""
    bad = []
    m, n, k = 9, 11, 13
    A, B, C = gi.random_problem(66, m, n, k, "i16")
    exp = numpy_gemm(A, B, C)
    Ap = np.full((m, k + 5), 12345, np.int16)
    Bp = np.full((k, n + 3), -777, np.int16)
    Cp = np.full((m, n + 7), -424242, np.int64)
    Ap[:, :k] = A
    Bp[:, :n] = B
    Cp[:, :n] = C
    oracle.gemm(Ap[:, :k], Bp[:, :n], Cp[:, :n], lib=lib)
    if not np.array_equal(Cp[:, :n], exp):
        bad.append("padded result")
    if not (Cp[:, n:] == -424242).all():
        bad.append("padding of C touched")
    return bad


def check_linearity(lib):
    bad = []
    m, n, k = 20, 30, 40
    A1, B, C = gi.random_problem(81, m, n, k, "i16", a_range=(-16384, 16383))
    A2, _, _ = gi.random_problem(82, m, n, k, "i16", a_range=(-16384, 16383))
    z = np.zeros((m, n), np.int64)
    lhs = _run(lib, (A1 + A2).astype(np.int16), B, z)
    rhs = _run(lib, A1, B, z) + _run(lib, A2, B, z)
    if not np.array_equal(lhs, rhs):
        bad.append("linear in A")
    B1, B2 = B // 2, B - B // 2
    if not np.array_equal(_run(lib, A1, B, z), _run(lib, A1, B1.astype(np.int16), z) + _run(lib, A1, B2.astype(np.int16), z)):
        bad.append("linear in B")
    if not np.array_equal(_run(lib, A1, B, C) - _run(lib, A1, B, z), C):
        bad.append("offset by C_in")
    return bad


def check_transpose(lib):
    m, n, k = 13, 29, 7
    A, B, C = gi.random_problem(91, m, n, k, "i16")
    X = _run(lib, A, B, C)
    Y = _run(lib, np.ascontiguousarray(B.T), np.ascontiguousarray(A.T), np.ascontiguousarray(C.T))
    return [] if np.array_equal(X, Y.T) else ["transpose identity (AB)^T = B^T A^T"]


# ---- the paper's micro-kernel output: C16 += srs(A*B, shift)  (gemm_oracle_i16_srs)
SRS_GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "srs_cases.json")


def _run_srs(lib, A, B, C, shift):
    X = C.copy()
    oracle.gemm_srs(A, B, X, shift, lib=lib)
    return X


def check_srs_golden(lib):
    """Worked examples (tests/golden/srs_cases.json): rounding, saturation, wrapping add."""
    bad = []
    with open(SRS_GOLDEN) as f:
        cases = json.load(f)["cases"]
    for c in cases:
        m, n, k = c["m"], c["n"], c["k"]
        A = np.array(c["A"], dtype=np.int16).reshape(m, k)
        B = np.array(c["B"], dtype=np.int16).reshape(k, n)
        C = np.array(c["C_in"], dtype=np.int16).reshape(m, n)
        E = np.array(c["C_out"], dtype=np.int16).reshape(m, n)
        got = _run_srs(lib, A, B, C, c["shift"])
        if not np.array_equal(got, E):
            bad.append(f"srs golden {c['name']}: got {got.tolist()} want {E.tolist()}")
    return bad


def check_srs_reduces_to_gemm(lib):
    """Shift 0 with sums inside int16: srs is the identity, so C16 + S taken modulo 2^16 must match
    the exact GEMM (numpy's integer matmul) -- on every entry, with values chosen so that no sum
    saturates."""
    bad = []
    for seed, (m, n, k) in enumerate(((3, 5, 7), (17, 9, 40), (40, 33, 64))):
        A = gi.uniform_int(700 + seed, (m, k), -11, 11, np.int16)
        B = gi.uniform_int(710 + seed, (k, n), -11, 11, np.int16)
        C = gi.uniform_int(720 + seed, (m, n), -32768, 32767, np.int16)
        S = np.matmul(A.astype(np.int64), B.astype(np.int64))
        assert np.abs(S).max() <= 32767
        want = ((C.astype(np.int64) + S) & 0xFFFF).astype(np.uint16).view(np.int16)
        if not np.array_equal(_run_srs(lib, A, B, C, 0), want):
            bad.append(f"srs shift 0 != exact GEMM mod 2^16 on {(m, n, k)}")
    return bad


def check_srs_closed_forms(lib):
    """All-ones operands give S = k on every entry: srs is then known in closed form."""
    bad = []
    for k, shift, want in ((5, 1, 3), (6, 2, 2), (7, 1, 4), (40000, 0, 32767), (40000, 1, 20000),
                           (65535, 1, 32767), (9, 3, 1), (12, 3, 2)):
        A = np.ones((2, k), np.int16)
        B = np.ones((k, 3), np.int16)
        got = _run_srs(lib, A, B, np.zeros((2, 3), np.int16), shift)
        if not (got == want).all():
            bad.append(f"srs all-ones k={k} shift={shift}: got {got[0, 0]} want {want}")
        got = _run_srs(lib, -A, B, np.zeros((2, 3), np.int16), shift)
        # -k/2^shift rounded half up: e.g. -2.5 -> -2; -40000 saturates at -32768
        wn = {(5, 1): -2, (6, 2): -1, (7, 1): -3, (40000, 0): -32768, (40000, 1): -20000,
              (65535, 1): -32767, (9, 3): -1, (12, 3): -1}[(k, shift)]
        if not (got == wn).all():
            bad.append(f"srs all-minus-ones k={k} shift={shift}: got {got[0, 0]} want {wn}")
    return bad


SRS_CHECKS = (check_srs_golden, check_srs_reduces_to_gemm, check_srs_closed_forms)


# ---- convolution through the lowered GEMM: Y += conv(X, Wt)  (gemm_oracle_conv2d_i16)
CONV_GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "conv_cases.json")


def _conv(lib, X, Wt, Y, R, S, ph, pw):
    Z = Y.copy()
    oracle.conv2d(X, Wt, Z, R, S, ph, pw, lib=lib)
    return Z


def check_conv_golden(lib):
    bad = []
    with open(CONV_GOLDEN) as f:
        cases = json.load(f)["cases"]
    for c in cases:
        N, H, W, Ci, Co, R, S, ph, pw = (c[x] for x in ("N", "H", "W", "Cin", "Cout", "R", "S", "pad_h", "pad_w"))
        Ho, Wo = H + 2 * ph - R + 1, W + 2 * pw - S + 1
        X = np.array(c["X"], np.int16).reshape(N, H, W, Ci)
        Wt = np.array(c["Wt"], np.int16).reshape(R * S * Ci, Co)
        Y = np.array(c["Y_in"], np.int64).reshape(N, Ho, Wo, Co)
        E = np.array(c["Y_out"], np.int64).reshape(N, Ho, Wo, Co)
        got = _conv(lib, X, Wt, Y, R, S, ph, pw)
        if not np.array_equal(got, E):
            bad.append(f"conv golden {c['name']}: got {got.ravel().tolist()} want {E.ravel().tolist()}")
    return bad


def check_conv_1x1_is_gemm(lib):
    """A 1x1 convolution is the GEMM of the pixels (N*H*W x Cin) by the weights: numpy's matmul."""
    bad = []
    for seed, (N, H, W, Ci, Co) in enumerate(((2, 3, 5, 4, 6), (1, 7, 2, 9, 3))):
        X = gi.uniform_int(730 + seed, (N, H, W, Ci), -32768, 32767, np.int16)
        Wt = gi.uniform_int(740 + seed, (Ci, Co), -32768, 32767, np.int16)
        Y = gi.uniform_int(750 + seed, (N, H, W, Co), -(1 << 40), 1 << 40, np.int64)
        want = Y + np.matmul(X.reshape(-1, Ci).astype(np.int64), Wt.astype(np.int64)).reshape(N, H, W, Co)
        if not np.array_equal(_conv(lib, X, Wt, Y, 1, 1, 0, 0), want):
            bad.append(f"conv 1x1 != GEMM on {(N, H, W, Ci, Co)}")
    return bad


def check_conv_delta_kernels(lib):
    """A kernel that is 1 at one tap and the identity across channels copies the input, shifted by
    that tap's offset, with zeros where the shifted pixel lies outside the image."""
    bad = []
    N, H, W, C = 2, 5, 4, 3
    X = gi.uniform_int(760, (N, H, W, C), -32768, 32767, np.int16)
    Xp = np.pad(X.astype(np.int64), ((0, 0), (1, 1), (1, 1), (0, 0)))
    for r in range(3):
        for s in range(3):
            Wt = np.zeros((9 * C, C), np.int16)
            for c in range(C):
                Wt[(r * 3 + s) * C + c, c] = 1
            want = Xp[:, r:r + H, s:s + W, :]  # Y[h][w] = X[h + r - 1][w + s - 1], zero outside
            got = _conv(lib, X, Wt, np.zeros((N, H, W, C), np.int64), 3, 3, 1, 1)
            if not np.array_equal(got, want):
                bad.append(f"conv delta at tap ({r},{s})")
    return bad


def check_conv_im2col_lowering(lib):
    """The IM2COL transform (Section 2 of the paper): build the lowered matrix element by element
    and multiply it by the weights with numpy's integer matmul."""
    bad = []
    for seed, (N, H, W, Ci, Co, R, S, ph, pw) in enumerate(((1, 4, 5, 2, 3, 3, 3, 1, 1),
                                                            (2, 3, 6, 3, 2, 2, 3, 0, 1))):
        Ho, Wo = H + 2 * ph - R + 1, W + 2 * pw - S + 1
        X = gi.uniform_int(770 + seed, (N, H, W, Ci), -32768, 32767, np.int16)
        Wt = gi.uniform_int(780 + seed, (R * S * Ci, Co), -32768, 32767, np.int16)
        low = np.zeros((N * Ho * Wo, R * S * Ci), np.int64)
        for n in range(N):
            for ho in range(Ho):
                for wo in range(Wo):
                    for r in range(R):
                        for s in range(S):
                            h, w = ho + r - ph, wo + s - pw
                            if 0 <= h < H and 0 <= w < W:
                                for c in range(Ci):
                                    low[(n * Ho + ho) * Wo + wo, (r * S + s) * Ci + c] = X[n, h, w, c]
        want = np.matmul(low, Wt.astype(np.int64)).reshape(N, Ho, Wo, Co)
        if not np.array_equal(_conv(lib, X, Wt, np.zeros((N, Ho, Wo, Co), np.int64), R, S, ph, pw), want):
            bad.append(f"conv != IM2COL lowering on {(N, H, W, Ci, Co, R, S, ph, pw)}")
    return bad


CONV_CHECKS = (check_conv_golden, check_conv_1x1_is_gemm, check_conv_delta_kernels, check_conv_im2col_lowering)

# ---- the int4 variant: C32 += A*B with operands packed two to a byte  (gemm_oracle_i4)
I4_GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "i4_cases.json")


def _run_i4(lib, Ap, Bp, C, k):
    X = C.copy()
    oracle.gemm_i4(Ap, Bp, X, k, lib=lib)
    return X


def unpack_nibbles_bigint(rows, cols):
    """Signed 4-bit values read back from packed bytes with Python integers, written independently
    of both the oracle and the packer: bit 4*(c%2) of byte c//2, sign from bit 3."""
    out = []
    for r in rows:
        vals = []
        for c in range(cols):
            nib = (int(r[c // 2]) >> (4 * (c % 2))) & 15
            vals.append(nib - 16 if nib & 8 else nib)
        out.append(vals)
    return np.array(out, dtype=np.int64).reshape(len(rows), cols)


def check_i4_golden(lib):
    """Worked examples (tests/golden/i4_cases.json): nibble order, two's complement, odd k and n,
    row padding, wrap-around modulo 2^32."""
    bad = []
    with open(I4_GOLDEN) as f:
        cases = json.load(f)["cases"]
    for c in cases:
        m, n, k = c["m"], c["n"], c["k"]
        Ap = np.array(c["A"], np.uint8).reshape(m, c["lda"])
        Bp = np.array(c["B"], np.uint8).reshape(k, c["ldb"])
        C = np.array(c["C_in"], np.int32).reshape(m, n)
        E = np.array(c["C_out"], np.int32).reshape(m, n)
        got = _run_i4(lib, Ap[:, :(k + 1) // 2] if c["lda"] > (k + 1) // 2 else Ap,
                      Bp[:, :(n + 1) // 2] if c["ldb"] > (n + 1) // 2 else Bp, C, k)
        if not np.array_equal(got, E):
            bad.append(f"i4 golden {c['name']}: got {got.tolist()} want {E.tolist()}")
    return bad


def check_i4_bruteforce(lib, shapes=((1, 1, 1), (2, 3, 5), (5, 7, 9), (3, 8, 17), (8, 1, 33))):
    """Tiny shapes against Python integers on the values unpacked independently from the bytes;
    the spare nibble of odd rows and the padding bytes hold a non-zero pattern."""
    bad = []
    for idx, (m, n, k) in enumerate(shapes):
        A, B, C = gi.random_problem(7400 + idx, m, n, k, "i4")
        Ap = gi.pack_nibbles(A, ld=(k + 1) // 2 + 2, pad=0x9B)
        Bp = gi.pack_nibbles(B, ld=(n + 1) // 2 + 1, pad=0x6E)
        Av = unpack_nibbles_bigint(Ap, k)
        Bv = unpack_nibbles_bigint(Bp, n)
        if not (np.array_equal(Av, A) and np.array_equal(Bv, B)):
            bad.append(f"i4 packer does not store the documented format ({m}x{n}x{k})")
        exp = bigint_gemm(Av, Bv, C.astype(np.int64), 32).astype(np.int32)
        got = _run_i4(lib, Ap[:, :(k + 1) // 2], Bp[:, :(n + 1) // 2], C, k)
        if not np.array_equal(got, exp):
            bad.append(f"i4 bruteforce {m}x{n}x{k}")
    return bad


def check_i4_matches_i8(lib, shapes=((33, 20, 71), (64, 65, 128), (7, 130, 301))):
    """A special case that reduces to a pinned routine: the int4 GEMM of values in [-8, 7] equals the
    int8 GEMM of the same values (and numpy's exact matmul), padded rows and all."""
    bad = []
    for idx, (m, n, k) in enumerate(shapes):
        A, B, C = gi.random_problem(7500 + idx, m, n, k, "i4")
        Ap = gi.pack_nibbles(A, ld=(k + 1) // 2 + 3, pad=0x7F)
        Bp = gi.pack_nibbles(B, ld=(n + 1) // 2 + 5, pad=0x81)
        got = _run_i4(lib, Ap[:, :(k + 1) // 2], Bp[:, :(n + 1) // 2], C, k)
        if not np.array_equal(got, _run(lib, A, B, C)):
            bad.append(f"i4 != i8 GEMM of the same values on {(m, n, k)}")
        if not np.array_equal(got, numpy_gemm(A, B, C)):
            bad.append(f"i4 != numpy matmul on {(m, n, k)}")
    return bad


def check_i4_closed_forms(lib):
    """Constant operands: every entry of C gains k*a*b."""
    bad = []
    for k in (1, 2, 7, 300):
        for a, b in ((-8, -8), (7, -8), (7, 7), (-1, 1)):
            m, n = 3, 5
            Ap = gi.pack_nibbles(np.full((m, k), a, np.int8))
            Bp = gi.pack_nibbles(np.full((k, n), b, np.int8))
            got = _run_i4(lib, Ap, Bp, np.zeros((m, n), np.int32), k)
            if not (got == k * a * b).all():
                bad.append(f"i4 constant a={a} b={b} k={k}: got {got[0, 0]} want {k * a * b}")
    return bad


I4_CHECKS = (check_i4_golden, check_i4_bruteforce, check_i4_matches_i8, check_i4_closed_forms)

ALL_CHECKS = (check_golden, check_extreme_bruteforce, check_closed_forms, check_identity_permutation,
              check_blocked, check_padding, check_linearity, check_transpose, check_numpy) + SRS_CHECKS + CONV_CHECKS + I4_CHECKS


def pin_failures(lib, bruteforce_shapes=None):
    bad = []
    for chk in ALL_CHECKS:
        try:
            bad += chk(lib)
        except Exception as e:  # a crash of a mutant counts as detected
            bad.append(f"{chk.__name__} raised {type(e).__name__}: {e}")
    try:
        bad += check_bruteforce(lib, shapes=bruteforce_shapes)
    except Exception as e:
        bad.append(f"bruteforce raised {e}")
    return bad
