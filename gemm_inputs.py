"""Seeded synthetic inputs for the exact integer GEMM  C += A*B.

This module only draws numbers.  It holds none of the GEMM arithmetic, and it
is the one module shared by the CPU oracle's tests and the CUDA path's tests
and benchmark: both sides receive the same arrays from here.

Generator: SplitMix64 (G. L. Steele, D. Lea, C. H. Flood, "Fast splittable
pseudorandom number generators", OOPSLA 2014).  The state advances by the
golden-gamma constant 0x9E3779B97F4A7C15 and each output is the state passed
through the published 64-bit finaliser (xor-shift 30, multiply, xor-shift 27,
multiply, xor-shift 31).  Element e of a stream seeded with s is output number
e+1 of a SplitMix64 started at state s, i.e. mix(s + (e+1)*gamma), so any
element can be drawn independently of the others (counter-based).

Value mapping: an integer uniform on [lo, hi] is lo + (r mod (hi-lo+1)) for
the 64-bit draw r (the bias is below 2^-40 for the ranges used here).  The
im2col activation matrix of the 3x3-convolution workload is 50% exact zeros:
the top bit of r decides zero / non-zero and the non-zero branch takes
r mod 4096, so P(value == 0) = 0.5 + 0.5/4096.

The workloads (matrix shapes, operand types and value distributions) are
those of the GEMM problem of Section 4.1 of the paper at the sizes the
benchmark studies; the paper itself uses INT16 operands (Section 6.1) and
lowers convolutions to GEMM through IM2COL/IM2ROW (Sections 2, 4.2, 5.1).
The int4 workload is the lower-precision point the paper leaves to future
work (Section 6.1).
Matrix X of workload w is drawn from stream 4*seed_w + {A: 0, B: 1, C: 2}.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

GAMMA = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)
_CHUNK = 1 << 22


def splitmix64(seed: int, start: int, count: int) -> np.ndarray:
    """Outputs start+1 .. start+count of SplitMix64 seeded with `seed` (uint64)."""
    seed = np.uint64(seed & 0xFFFFFFFFFFFFFFFF)
    out = np.empty(count, dtype=np.uint64)
    with np.errstate(over="ignore"):
        for c0 in range(0, count, _CHUNK):
            c1 = min(count, c0 + _CHUNK)
            idx = np.arange(start + c0 + 1, start + c1 + 1, dtype=np.uint64)
            z = seed + idx * GAMMA
            z = (z ^ (z >> np.uint64(30))) * _M1
            z = (z ^ (z >> np.uint64(27))) * _M2
            out[c0:c1] = z ^ (z >> np.uint64(31))
    return out


def uniform_int(seed: int, shape, lo: int, hi: int, dtype) -> np.ndarray:
    """Integers uniform on [lo, hi] (inclusive), drawn element-wise in C order."""
    n = int(np.prod(shape)) if len(shape) else 1
    r = splitmix64(seed, 0, n)
    span = np.uint64(hi - lo + 1)
    v = (r % span).astype(np.int64) + lo
    return v.astype(dtype).reshape(shape)


def half_zero_uniform(seed: int, shape, hi: int, dtype) -> np.ndarray:
    """50% exact zeros (top bit of the draw), else uniform on [0, hi]."""
    n = int(np.prod(shape))
    r = splitmix64(seed, 0, n)
    nonzero = (r >> np.uint64(63)) == np.uint64(1)
    v = (r % np.uint64(hi + 1)).astype(np.int64)
    v[~nonzero] = 0
    return v.astype(dtype).reshape(shape)


@dataclass(frozen=True)
class Workload:
    """One benchmark workload: C (m x n) += A (m x k) * B (k x n)."""
    name: str
    kind: str          # "i16" (int16 operands, int64 C), "i8" (int8, int32 C) or "i4" (int4 values held
                       # one per int8 element, stored packed two to a byte by pack_nibbles; int32 C)
    m: int
    n: int
    k: int
    seed: int
    a_dist: tuple      # ("uniform", lo, hi) or ("half_zero", hi)
    b_dist: tuple
    c_dist: tuple      # ("uniform", lo, hi) or ("zero",)
    note: str

    @property
    def op_dtype(self):
        return np.int16 if self.kind == "i16" else np.int8

    @property
    def c_dtype(self):
        return np.int64 if self.kind == "i16" else np.int32

    @property
    def ops(self) -> int:
        """Algorithmic integer operations, 2*m*n*k (one multiply + one add per MAC)."""
        return 2 * self.m * self.n * self.k


FULL16 = ("uniform", -32768, 32767)

WORKLOADS = {
    "i16_256": Workload("i16_256", "i16", 256, 256, 256, 1001, FULL16, FULL16,
                        ("uniform", -(1 << 20), 1 << 20),
                        "int16 GEMM 256^3, full-range operands, C uniform in [-2^20, 2^20]"),
    "i8_4096": Workload("i8_4096", "i8", 4096, 4096, 4096, 1002, ("uniform", -128, 127),
                        ("uniform", -128, 127), ("zero",),
                        "int8 GEMM 4096^3, s8 operands uniform in [-128, 127], C int32 = 0"),
    "conv3x3_im2col": Workload("conv3x3_im2col", "i16", 100352, 64, 576, 1003, ("half_zero", 4095),
                               ("uniform", -2048, 2047), ("zero",),
                               "im2col GEMM of a 3x3/s1/p1 conv, batch 32, 56x56 output, 64->64 channels"),
    "i16_8192": Workload("i16_8192", "i16", 8192, 8192, 8192, 1004, FULL16, FULL16, ("zero",),
                         "int16 GEMM 8192^3, full-range operands, C int64 = 0"),
    "skinny_8x4096x4096": Workload("skinny_8x4096x4096", "i16", 8, 4096, 4096, 1005, FULL16, FULL16,
                                   ("zero",), "batch-8 fully-connected layer, m=8, n=k=4096"),
    "i4_8192": Workload("i4_8192", "i4", 8192, 8192, 8192, 1007, ("uniform", -8, 7), ("uniform", -8, 7), ("zero",),
                        "int4 GEMM 8192^3 (the lower-precision point), operands uniform in [-8, 7], C int32 = 0"),
}


def _draw(seed: int, shape, dist, dtype) -> np.ndarray:
    if dist[0] == "uniform":
        return uniform_int(seed, shape, dist[1], dist[2], dtype)
    if dist[0] == "half_zero":
        return half_zero_uniform(seed, shape, dist[1], dtype)
    if dist[0] == "zero":
        return np.zeros(shape, dtype=dtype)
    raise ValueError(dist)


def make_inputs(w: Workload, rows: slice | None = None):
    """(A, B, C) as contiguous row-major numpy arrays for workload w.

    `rows` restricts A and C to a slice of rows (the same values those rows have
    in the full problem), which is how bounded samples of a large workload are
    drawn for the CPU baseline.
    """
    r0, r1 = (0, w.m) if rows is None else (rows.start or 0, rows.stop if rows.stop is not None else w.m)
    mr = r1 - r0
    A = _draw_rows(4 * w.seed + 0, w.m, w.k, r0, mr, w.a_dist, w.op_dtype)
    B = _draw(4 * w.seed + 1, (w.k, w.n), w.b_dist, w.op_dtype)
    C = _draw_rows(4 * w.seed + 2, w.m, w.n, r0, mr, w.c_dist, w.c_dtype)
    return A, B, C


def _draw_rows(seed: int, m: int, cols: int, r0: int, mr: int, dist, dtype) -> np.ndarray:
    """Rows r0 .. r0+mr of an m x cols matrix drawn element-wise in C order."""
    if dist[0] == "zero":
        return np.zeros((mr, cols), dtype=dtype)
    n = mr * cols
    r = splitmix64(seed, r0 * cols, n)
    if dist[0] == "uniform":
        v = (r % np.uint64(dist[2] - dist[1] + 1)).astype(np.int64) + dist[1]
    elif dist[0] == "half_zero":
        v = (r % np.uint64(dist[1] + 1)).astype(np.int64)
        v[(r >> np.uint64(63)) == np.uint64(0)] = 0
    else:
        raise ValueError(dist)
    return v.astype(dtype).reshape(mr, cols)


def pack_nibbles(v: np.ndarray, ld: int | None = None, pad: int = 0) -> np.ndarray:
    """Store signed 4-bit values two to a byte (the int4 operand format).

    v: integer array (rows, cols) with values in [-8, 7].  Element (r, c) goes to byte c//2 of row
    r, in the low nibble when c is even and the high nibble when c is odd, as its two's-complement
    bit pattern (v & 15).  Rows are `ld` bytes apart (default ceil(cols/2)); the bytes past the
    packed width and the spare high nibble of an odd-width row hold `pad`'s bit patterns.
    """
    rows, cols = v.shape
    width = (cols + 1) // 2
    ld = width if ld is None else ld
    if ld < width:
        raise ValueError("row pitch below the packed width")
    if v.size and (v.min() < -8 or v.max() > 7):
        raise ValueError("int4 values must lie in [-8, 7]")
    nib = (v.astype(np.int64) & 15).astype(np.uint8)
    if cols % 2:
        nib = np.concatenate([nib, np.full((rows, 1), pad & 15, np.uint8)], axis=1)
    out = np.full((rows, ld), pad & 0xFF, np.uint8)
    out[:, :width] = nib[:, 0::2] | (nib[:, 1::2] << np.uint8(4))
    return out


def random_problem(seed: int, m: int, n: int, k: int, kind: str = "i16",
                   a_range=None, b_range=None, c_range=None):
    """Arbitrary-shape seeded problem for tests (row-major, contiguous).

    kind "i4" draws int4 values in [-8, 7], held one per int8 element (pack_nibbles stores them).
    """
    op = np.int16 if kind == "i16" else np.int8
    cd = np.int64 if kind == "i16" else np.int32
    full = {"i16": (-32768, 32767), "i8": (-128, 127), "i4": (-8, 7)}[kind]
    a_range = a_range or full
    b_range = b_range or full
    c_range = c_range or ((-(1 << 40), 1 << 40) if kind == "i16" else (-(1 << 30), 1 << 30))
    A = uniform_int(4 * seed + 0, (m, k), a_range[0], a_range[1], op)
    B = uniform_int(4 * seed + 1, (k, n), b_range[0], b_range[1], op)
    C = uniform_int(4 * seed + 2, (m, n), c_range[0], c_range[1], cd)
    return A, B, C
