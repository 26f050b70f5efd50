"""CPU oracle for the exact integer GEMM  C += A*B  (test infrastructure only).

Only the tests, the smoke check and the benchmark's CPU-baseline leg may
import this package.  The product path (the CUDA library and its binding)
never loads it, and it shares no code with that path.

The arithmetic lives in `gemm_oracle.c` (plain triple loop, 64-bit modular
sums; the GEMM definition of Section 4.1 of the paper).  This module compiles
it with the host C compiler and calls it through ctypes on numpy arrays.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "gemm_oracle.c")
_LIB = os.path.join(_HERE, "libgemm_oracle.so")
_lib = None


def build(force: bool = False, src: str = _SRC, out: str = _LIB, extra=()) -> str:
    """Compile the oracle into a shared object (OpenMP when available)."""
    if not force and os.path.exists(out) and os.path.getmtime(out) >= os.path.getmtime(src):
        return out
    base = ["gcc", "-O2", "-std=c11", "-shared", "-fPIC", *extra, src, "-o", out]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True, capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    return out


def load(path: str | None = None):
    """Load (building first if needed) the oracle library."""
    global _lib
    if path is not None:
        return _bind(ctypes.CDLL(path))
    if _lib is None:
        _lib = _bind(ctypes.CDLL(build()))
    return _lib


def _bind(lib):
    i64, vp = ctypes.c_int64, ctypes.c_void_p
    for name in ("gemm_oracle_i16", "gemm_oracle_i8"):
        f = getattr(lib, name)
        f.argtypes = [i64, i64, i64, vp, i64, vp, i64, vp, i64, ctypes.c_int]
        f.restype = ctypes.c_int
    lib.gemm_oracle_i4.argtypes = [i64, i64, i64, vp, i64, vp, i64, vp, i64, ctypes.c_int]
    lib.gemm_oracle_i4.restype = ctypes.c_int
    lib.gemm_oracle_i16_srs.argtypes = [i64, i64, i64, vp, i64, vp, i64, vp, i64, ctypes.c_int, ctypes.c_int]
    lib.gemm_oracle_i16_srs.restype = ctypes.c_int
    lib.gemm_oracle_conv2d_i16.argtypes = [i64] * 9 + [vp, vp, vp, ctypes.c_int]
    lib.gemm_oracle_conv2d_i16.restype = ctypes.c_int
    lib.gemm_oracle_max_threads.restype = ctypes.c_int
    return lib


def _ptr(x: np.ndarray):
    return ctypes.c_void_p(x.ctypes.data) if x.size else ctypes.c_void_p(0)


def _ld(x: np.ndarray, itemsize: int) -> int:
    if x.ndim != 2:
        raise ValueError("oracle operands must be 2-D")
    rows, cols = x.shape
    if x.size == 0 or rows == 1:
        return max(cols, 1)
    if (cols > 1 and x.strides[1] != itemsize) or x.strides[0] % itemsize or x.strides[0] < cols * itemsize:
        raise ValueError("oracle operands must be row-major with unit column stride")
    return max(x.strides[0] // itemsize, cols, 1)


def gemm(A: np.ndarray, B: np.ndarray, C: np.ndarray, nthreads: int = 1, lib=None) -> np.ndarray:
    """In place: C += A @ B, exactly (int16 -> int64 mod 2^64, int8 -> int32 mod 2^32).

    A, B, C may be row-major views with padded rows (leading dimension =
    row stride); C is returned for convenience.
    """
    lib = lib or load()
    if A.dtype == np.int16:
        fn, cd = lib.gemm_oracle_i16, np.int64
        if B.dtype != np.int16 or C.dtype != np.int64:
            raise TypeError("int16 GEMM wants int16 A, B and an int64 C")
    elif A.dtype == np.int8:
        fn, cd = lib.gemm_oracle_i8, np.int32
        if B.dtype != np.int8 or C.dtype != np.int32:
            raise TypeError("int8 GEMM wants int8 A, B and an int32 C")
    else:
        raise TypeError(f"unsupported operand type {A.dtype}")
    m, k = A.shape
    k2, n = B.shape
    if k2 != k or C.shape != (m, n):
        raise ValueError(f"shape mismatch: A {A.shape}, B {B.shape}, C {C.shape}")
    rc = fn(m, n, k, _ptr(A), _ld(A, A.itemsize), _ptr(B), _ld(B, B.itemsize),
            _ptr(C), _ld(C, C.itemsize), int(nthreads))
    if rc != 0:
        raise ValueError(f"oracle rejected the arguments (rc={rc})")
    return C


def gemm_i4(Ap: np.ndarray, Bp: np.ndarray, C: np.ndarray, k: int, nthreads: int = 1, lib=None) -> np.ndarray:
    """In place: C (int32) += A @ B modulo 2^32, A and B signed 4-bit values packed two to a byte.

    Ap: uint8 (m, >= ceil(k/2)) holding A's rows, element (i, p) in byte p//2 (low nibble for even
    p, high nibble for odd p, two's complement); Bp: uint8 (k, >= ceil(n/2)) holding B's rows the
    same way along j.  Row pitches may exceed the packed width (padding is never read).
    """
    lib = lib or load()
    if Ap.dtype != np.uint8 or Bp.dtype != np.uint8 or C.dtype != np.int32:
        raise TypeError("gemm_i4 takes uint8 packed A and B and an int32 C")
    m, n = C.shape
    if Ap.shape[0] != m or Bp.shape[0] != k or Ap.shape[1] < (k + 1) // 2 or Bp.shape[1] < (n + 1) // 2:
        raise ValueError(f"shape mismatch: packed A {Ap.shape}, packed B {Bp.shape}, C {C.shape}, k {k}")
    lda = _ld(Ap, 1) if m else max(1, (k + 1) // 2)
    ldb = _ld(Bp, 1) if k else max(1, (n + 1) // 2)
    rc = lib.gemm_oracle_i4(m, n, k, _ptr(Ap), lda, _ptr(Bp), ldb, _ptr(C), _ld(C, 4), int(nthreads))
    if rc != 0:
        raise ValueError(f"oracle rejected the arguments (rc={rc})")
    return C


def gemm_srs(A: np.ndarray, B: np.ndarray, C: np.ndarray, shift: int, nthreads: int = 1, lib=None) -> np.ndarray:
    """In place: C (int16) = wrap16(C + sat16(round_half_up(A @ B / 2^shift))), the paper's
    shift-round-saturate micro-kernel output (see gemm_oracle.c for the readings)."""
    lib = lib or load()
    if A.dtype != np.int16 or B.dtype != np.int16 or C.dtype != np.int16:
        raise TypeError("gemm_srs takes int16 A, B and C")
    m, k = A.shape
    k2, n = B.shape
    if k2 != k or C.shape != (m, n):
        raise ValueError(f"shape mismatch: A {A.shape}, B {B.shape}, C {C.shape}")
    rc = lib.gemm_oracle_i16_srs(m, n, k, _ptr(A), _ld(A, 2), _ptr(B), _ld(B, 2), _ptr(C), _ld(C, 2),
                                 int(shift), int(nthreads))
    if rc != 0:
        raise ValueError("oracle rejected the arguments")
    return C


def conv2d(X: np.ndarray, Wt: np.ndarray, Y: np.ndarray, R: int, S: int, pad_h: int, pad_w: int,
           nthreads: int = 1, lib=None) -> np.ndarray:
    """In place: Y += conv(X, Wt), stride 1, zero padding (see gemm_oracle.c).

    X: int16 (N, H, W, Cin); Wt: int16 (R*S*Cin, Cout) in (r, s, c) row order; Y: int64
    (N, Ho, Wo, Cout) with Ho = H + 2*pad_h - R + 1, Wo = W + 2*pad_w - S + 1.  All C-contiguous.
    """
    lib = lib or load()
    N, H, W, Cin = X.shape
    K, Cout = Wt.shape
    Ho, Wo = H + 2 * pad_h - R + 1, W + 2 * pad_w - S + 1
    if X.dtype != np.int16 or Wt.dtype != np.int16 or Y.dtype != np.int64:
        raise TypeError("conv2d takes int16 X and Wt and an int64 Y")
    if K != R * S * Cin or Y.shape != (N, Ho, Wo, Cout):
        raise ValueError(f"shape mismatch: X {X.shape}, Wt {Wt.shape}, Y {Y.shape}")
    for t in (X, Wt, Y):
        if not t.flags.c_contiguous:
            raise ValueError("conv2d operands must be C-contiguous")
    rc = lib.gemm_oracle_conv2d_i16(N, H, W, Cin, Cout, R, S, pad_h, pad_w, _ptr(X), _ptr(Wt), _ptr(Y),
                                    int(nthreads))
    if rc != 0:
        raise ValueError("oracle rejected the arguments")
    return Y


def max_threads() -> int:
    return int(load().gemm_oracle_max_threads())


def host_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:  # pragma: no cover
        return os.cpu_count() or 1
