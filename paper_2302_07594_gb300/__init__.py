"""Exact integer GEMM (C += A*B) on NVIDIA GB300: Python binding of libgemmi.

The C library (include/gemmi.h, built from csrc/ by `build()`) does all the
work on the GPU; this module only marshals arguments through ctypes.  There is
no CPU fallback: if the library is missing, every call raises.

    gemm_i16(A, B, C)       torch CUDA tensors: int16 A (m x k), B (k x n), int64 C (m x n)
    gemm_i8(A, B, C)        torch CUDA tensors: int8 A, B, int32 C
    gemm_i4(A, B, C, k)     torch CUDA tensors: uint8 A, B holding int4 values two to a byte, int32 C
    gemm_i16_host(A, B, C)  numpy arrays (host memory): the library copies in and out
    gemm_i8_host(A, B, C), gemm_i4_host(A, B, C, k)
    pack_b_i16 / pack_b_i8 / pack_b_i4, gemm_*_packed   weights split once, reused by every call
    gemm_i16_srs, conv2d_i16, gemm_i16_noalloc          the other entry points of include/gemmi.h

Matrices are row-major with unit column stride; a row stride larger than the
row length (padding) is passed as the leading dimension.  C is updated in
place: C += A @ B, bit-exactly (modulo 2^64 for int64 C, 2^32 for int32 C).
The GEMM is the one of Section 4.1 of the paper; see include/gemmi.h.
"""
from __future__ import annotations

import ctypes
import os

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libgemmi.so")

OK, EINVAL, ENOMEM, ECUDA, ETIMEOUT, EARCH = 0, 1, 2, 3, 4, 5
OPT_SKINNY_MAX_M, OPT_WAIT_TIMEOUT_US, OPT_SKINNY_KSPLIT = 1, 2, 3
OPT_TC_CHUNK_SCALE, OPT_TC_GROUP_M, OPT_TC_L2_HINTS, OPT_FUSED_MAX_N, OPT_TC_PAIR = 4, 5, 6, 7, 8
OPT_SMALL_MAX_MACS, OPT_KARATSUBA, OPT_SPLIT_AHEAD, OPT_CONV_ROWS = 9, 10, 11, 12
EXPORTED = ("gemm_i16", "gemm_i16_ex", "gemm_i8", "gemm_i8_ex", "gemm_i16_host", "gemm_i8_host",
            "gemmi_set_stream", "gemmi_last_error", "gemmi_device_status", "gemmi_device_status_stream",
            "gemmi_device_status_detail", "gemmi_noalloc_selftest_wait_timeout", "gemmi_stream_read_probe",
            "gemmi_release_workspace", "gemmi_workspace_bytes", "gemmi_set_option", "gemmi_get_option",
            "gemmi_selftest_wait_timeout", "gemmi_kernel_timing", "gemmi_kernel_time", "gemmi_version",
            "gemm_i16_noalloc", "gemmi_pack_b_i16", "gemmi_pack_b_i8", "gemm_i16_packed", "gemm_i8_packed",
            "gemmi_packed_b_free", "gemmi_packed_b_k", "gemmi_packed_b_n", "gemm_i16_srs", "gemm_i16_srs_ex", "gemmi_conv2d_i16",
            "gemm_i4", "gemm_i4_ex", "gemmi_pack_b_i4", "gemm_i4_packed", "gemm_i4_host")
NOALLOC_SCRATCH_BYTES = 32 * 1024 * 1024
KERNEL_SPLIT, KERNEL_TC_I16, KERNEL_TC_I8, KERNEL_SKINNY, KERNEL_FUSED_I16, KERNEL_SRS = 0, 1, 2, 3, 4, 5
KERNEL_TC_PAIR_I16, KERNEL_TC_PAIR_I8, KERNEL_TC_PAIR_I4, KERNEL_ADD_I32, KERNEL_CONVERT_I4 = 6, 7, 8, 9, 10
KERNEL_TC_KARATSUBA, KERNEL_TC_PAIR_I16_AHEAD, KERNEL_CONV_ROWS = 11, 12, 13
KERNELS = (("split", KERNEL_SPLIT), ("tc_i16", KERNEL_TC_I16), ("tc_i8", KERNEL_TC_I8), ("skinny", KERNEL_SKINNY),
           ("fused_i16", KERNEL_FUSED_I16), ("srs", KERNEL_SRS), ("tc_pair_i16", KERNEL_TC_PAIR_I16),
           ("tc_pair_i8", KERNEL_TC_PAIR_I8), ("tc_pair_i4", KERNEL_TC_PAIR_I4), ("add_i32", KERNEL_ADD_I32),
           ("convert_i4", KERNEL_CONVERT_I4), ("tc_karatsuba", KERNEL_TC_KARATSUBA),
           ("tc_pair_i16_ahead", KERNEL_TC_PAIR_I16_AHEAD), ("conv_rows", KERNEL_CONV_ROWS))

_lib = None


class GemmiError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"gemmi error {code}: {msg}")
        self.code = code


def build(force: bool = False) -> str:
    from . import _build
    return _build.build(force=force)


def lib():
    """The loaded C library (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"libgemmi.so not found at {LIB_PATH}: build it first "
                               "(paper_2302_07594_gb300.build() or __graft_entry__.build())")
        L = ctypes.CDLL(LIB_PATH)
        i64, vp = ctypes.c_int64, ctypes.c_void_p
        core = [i64, i64, i64, vp, i64, vp, i64, vp, i64]
        for name in ("gemm_i16", "gemm_i8", "gemm_i16_host", "gemm_i8_host", "gemm_i4", "gemm_i4_host"):
            getattr(L, name).argtypes = core
            getattr(L, name).restype = ctypes.c_int
        for name in ("gemm_i16_ex", "gemm_i8_ex", "gemm_i16_noalloc", "gemm_i4_ex"):
            getattr(L, name).argtypes = core + [vp]
            getattr(L, name).restype = ctypes.c_int
        L.gemm_i16_srs.argtypes = core + [ctypes.c_int]
        L.gemm_i16_srs.restype = ctypes.c_int
        L.gemm_i16_srs_ex.argtypes = core + [ctypes.c_int, vp]
        L.gemm_i16_srs_ex.restype = ctypes.c_int
        L.gemmi_conv2d_i16.argtypes = [i64] * 9 + [vp, vp, vp, vp]
        L.gemmi_conv2d_i16.restype = ctypes.c_int
        L.gemmi_set_stream.argtypes = [vp]
        L.gemmi_set_stream.restype = None
        L.gemmi_last_error.restype = ctypes.c_char_p
        L.gemmi_device_status.restype = ctypes.c_int
        L.gemmi_device_status_stream.argtypes = [vp]
        L.gemmi_device_status_stream.restype = ctypes.c_int
        L.gemmi_noalloc_selftest_wait_timeout.argtypes = [i64, vp]
        L.gemmi_noalloc_selftest_wait_timeout.restype = ctypes.c_int
        L.gemmi_stream_read_probe.argtypes = [i64, i64, vp, i64, vp]
        L.gemmi_stream_read_probe.restype = ctypes.c_int
        L.gemmi_device_status_detail.restype = ctypes.c_uint32
        L.gemmi_release_workspace.restype = ctypes.c_int
        L.gemmi_workspace_bytes.restype = ctypes.c_size_t
        L.gemmi_set_option.argtypes = [ctypes.c_int, i64]
        L.gemmi_set_option.restype = ctypes.c_int
        L.gemmi_get_option.argtypes = [ctypes.c_int]
        L.gemmi_get_option.restype = i64
        L.gemmi_selftest_wait_timeout.argtypes = [i64]
        L.gemmi_selftest_wait_timeout.restype = ctypes.c_int
        L.gemmi_kernel_timing.argtypes = [ctypes.c_int]
        L.gemmi_kernel_timing.restype = ctypes.c_int
        L.gemmi_kernel_time.argtypes = [ctypes.c_int, ctypes.POINTER(ctypes.c_double), ctypes.POINTER(i64)]
        L.gemmi_kernel_time.restype = ctypes.c_int
        L.gemmi_version.restype = ctypes.c_char_p
        for name in ("gemmi_pack_b_i16", "gemmi_pack_b_i8", "gemmi_pack_b_i4"):
            getattr(L, name).argtypes = [i64, i64, vp, i64, vp, ctypes.POINTER(vp)]
            getattr(L, name).restype = ctypes.c_int
        for name in ("gemm_i16_packed", "gemm_i8_packed", "gemm_i4_packed"):
            getattr(L, name).argtypes = [i64, vp, i64, vp, vp, i64, vp]
            getattr(L, name).restype = ctypes.c_int
        L.gemmi_packed_b_free.argtypes = [vp]
        L.gemmi_packed_b_free.restype = ctypes.c_int
        for name in ("gemmi_packed_b_k", "gemmi_packed_b_n"):
            getattr(L, name).argtypes = [vp]
            getattr(L, name).restype = i64
        _lib = L
    return _lib


def _check(rc: int):
    if rc != OK:
        raise GemmiError(rc, lib().gemmi_last_error().decode(errors="replace"))


def last_error() -> str:
    return lib().gemmi_last_error().decode(errors="replace")


# ------------------------------------------------------------------ torch (device) entry points
def _dev_ld(t, name):
    if t.dim() != 2:
        raise ValueError(f"{name} must be 2-D")
    rows, cols = t.shape
    if t.numel() == 0 or rows == 1:
        return max(cols, 1)
    if (cols > 1 and t.stride(1) != 1) or t.stride(0) < cols:
        raise ValueError(f"{name} must be row-major with unit column stride")
    return t.stride(0)


def _torch_call(fn_name, A, B, C, op_dtype, c_dtype, stream):
    import torch
    for t, nm, dt in ((A, "A", op_dtype), (B, "B", op_dtype), (C, "C", c_dtype)):
        if not isinstance(t, torch.Tensor) or not t.is_cuda:
            raise TypeError(f"{nm} must be a CUDA tensor")
        if t.dtype != dt:
            raise TypeError(f"{nm} must be {dt}, got {t.dtype}")
    if not (A.device == B.device == C.device):
        raise ValueError("A, B and C must be on the same device")
    m, k = A.shape
    k2, n = B.shape
    if k2 != k or tuple(C.shape) != (m, n):
        raise ValueError(f"shape mismatch: A {tuple(A.shape)}, B {tuple(B.shape)}, C {tuple(C.shape)}")
    if stream is None:
        stream = torch.cuda.current_stream(A.device)
    with torch.cuda.device(A.device):
        rc = getattr(lib(), fn_name)(m, n, k, A.data_ptr(), _dev_ld(A, "A"), B.data_ptr(), _dev_ld(B, "B"),
                                     C.data_ptr(), _dev_ld(C, "C"), stream.cuda_stream)
    _check(rc)
    return C


def gemm_i16(A, B, C, stream=None):
    """C += A @ B on the GPU: int16 A (m x k), int16 B (k x n), int64 C (m x n); exact modulo 2^64."""
    import torch
    return _torch_call("gemm_i16_ex", A, B, C, torch.int16, torch.int64, stream)


def gemm_i16_noalloc(A, B, C, stream=None):
    """gemm_i16 for callers that must not allocate device memory (see include/gemmi.h).

    Uses the library's fixed scratch array instead of a workspace; problems needing more
    than NOALLOC_SCRATCH_BYTES of limb planes raise GemmiError (EINVAL).  Calls that overlap
    on the GPU share that array and must be serialised by the caller.
    """
    import torch
    return _torch_call("gemm_i16_noalloc", A, B, C, torch.int16, torch.int64, stream)


def gemm_i16_srs(A, B, C, shift, stream=None):
    """The paper's micro-kernel output on the GPU: int16 C += srs(A @ B, shift).

    The exact int16 product is shifted right by `shift` (rounding half up), saturated to int16
    and added to C modulo 2^16 (see gemm_i16_srs in include/gemmi.h).  C is int16.
    """
    import torch
    for t, nm in ((A, "A"), (B, "B"), (C, "C")):
        if not isinstance(t, torch.Tensor) or not t.is_cuda:
            raise TypeError(f"{nm} must be a CUDA tensor")
        if t.dtype != torch.int16:
            raise TypeError(f"{nm} must be torch.int16, got {t.dtype}")
    if not (A.device == B.device == C.device):
        raise ValueError("A, B and C must be on the same device")
    m, k = A.shape
    k2, n = B.shape
    if k2 != k or tuple(C.shape) != (m, n):
        raise ValueError(f"shape mismatch: A {tuple(A.shape)}, B {tuple(B.shape)}, C {tuple(C.shape)}")
    if stream is None:
        stream = torch.cuda.current_stream(A.device)
    with torch.cuda.device(A.device):
        rc = lib().gemm_i16_srs_ex(m, n, k, A.data_ptr(), _dev_ld(A, "A"), B.data_ptr(), _dev_ld(B, "B"),
                                   C.data_ptr(), _dev_ld(C, "C"), int(shift), stream.cuda_stream)
    _check(rc)
    return C


def conv2d_i16(X, Wt, Y, R, S, pad_h, pad_w, stream=None):
    """Y += conv(X, Wt) on the GPU: a stride-1, zero-padded convolution through the lowered GEMM.

    X: int16 (N, H, W, Cin) NHWC; Wt: int16 (R*S*Cin, Cout), rows in (r, s, c) order; Y: int64
    (N, Ho, Wo, Cout) with Ho = H + 2*pad_h - R + 1, Wo = W + 2*pad_w - S + 1.  All CUDA tensors,
    C-contiguous.  See gemmi_conv2d_i16 in include/gemmi.h.
    """
    import torch
    for t, nm, dt in ((X, "X", torch.int16), (Wt, "Wt", torch.int16), (Y, "Y", torch.int64)):
        if not isinstance(t, torch.Tensor) or not t.is_cuda:
            raise TypeError(f"{nm} must be a CUDA tensor")
        if t.dtype != dt:
            raise TypeError(f"{nm} must be {dt}, got {t.dtype}")
        if not t.is_contiguous():
            raise ValueError(f"{nm} must be contiguous")
    if not (X.device == Wt.device == Y.device):
        raise ValueError("X, Wt and Y must be on the same device")
    N, H, W, Cin = X.shape
    K, Cout = Wt.shape
    Ho, Wo = H + 2 * pad_h - R + 1, W + 2 * pad_w - S + 1
    if K != R * S * Cin or tuple(Y.shape) != (N, Ho, Wo, Cout):
        raise ValueError(f"shape mismatch: X {tuple(X.shape)}, Wt {tuple(Wt.shape)}, Y {tuple(Y.shape)}")
    if stream is None:
        stream = torch.cuda.current_stream(X.device)
    with torch.cuda.device(X.device):
        rc = lib().gemmi_conv2d_i16(N, H, W, Cin, Cout, R, S, pad_h, pad_w, X.data_ptr(), Wt.data_ptr(),
                                    Y.data_ptr(), stream.cuda_stream)
    _check(rc)
    return Y


def gemm_i8(A, B, C, stream=None):
    """C += A @ B on the GPU: int8 A, int8 B, int32 C; exact modulo 2^32."""
    import torch
    return _torch_call("gemm_i8_ex", A, B, C, torch.int8, torch.int32, stream)


def gemm_i4(A, B, C, k, stream=None):
    """C += A @ B on the GPU for signed 4-bit A (m x k) and B (k x n) packed two to a byte; int32 C,
    exact modulo 2^32.

    A: uint8 CUDA tensor (m, >= ceil(k/2)), element (i, p) in byte p // 2 of row i (low nibble for
    even p, high for odd p, two's complement); B: uint8 (k, >= ceil(n/2)) packed the same way
    along its rows; C: int32 (m, n).  k is passed because an odd k leaves a spare nibble per row.
    """
    import torch
    for t, nm, dt in ((A, "A", torch.uint8), (B, "B", torch.uint8), (C, "C", torch.int32)):
        if not isinstance(t, torch.Tensor) or not t.is_cuda:
            raise TypeError(f"{nm} must be a CUDA tensor")
        if t.dtype != dt:
            raise TypeError(f"{nm} must be {dt}, got {t.dtype}")
    if not (A.device == B.device == C.device):
        raise ValueError("A, B and C must be on the same device")
    m, n = C.shape
    k = int(k)
    if A.dim() != 2 or B.dim() != 2 or A.shape[0] != m or B.shape[0] != k or A.shape[1] < (k + 1) // 2 \
            or B.shape[1] < (n + 1) // 2:
        raise ValueError(f"shape mismatch: packed A {tuple(A.shape)}, packed B {tuple(B.shape)}, C {tuple(C.shape)}, k {k}")
    if stream is None:
        stream = torch.cuda.current_stream(A.device)
    with torch.cuda.device(A.device):
        rc = lib().gemm_i4_ex(m, n, k, A.data_ptr(), _dev_ld(A, "A"), B.data_ptr(), _dev_ld(B, "B"),
                              C.data_ptr(), _dev_ld(C, "C"), stream.cuda_stream)
    _check(rc)
    return C


# ------------------------------------------------------------------ pre-packed weights
class PackedB:
    """B (k x n) packed once on the device for repeated GEMMs (Section 5.1: weights are packed
    off-line, only activations at run time).  Frees its device memory when closed or collected."""

    def __init__(self, handle, kind, k, n, device):
        self._h = handle
        self.kind, self.k, self.n, self.device = kind, k, n, device

    @property
    def handle(self):
        if self._h is None:
            raise ValueError("packed operand was freed")
        return self._h

    def close(self):
        if self._h is not None:
            h, self._h = self._h, None
            _check(lib().gemmi_packed_b_free(h))

    def __del__(self):
        try:
            self.close()
        except Exception:  # interpreter shutdown
            pass


def _pack(fn_name, kind, B, dtype, stream, n=None):
    import torch
    if not isinstance(B, torch.Tensor) or not B.is_cuda or B.dtype != dtype:
        raise TypeError(f"B must be a CUDA {dtype} tensor")
    k, cols = B.shape
    n = cols if n is None else int(n)
    if cols < (n + 1) // 2:
        raise ValueError(f"packed B {tuple(B.shape)} is too narrow for n = {n}")
    if stream is None:
        stream = torch.cuda.current_stream(B.device)
    out = ctypes.c_void_p(0)
    with torch.cuda.device(B.device):
        rc = getattr(lib(), fn_name)(k, n, B.data_ptr(), _dev_ld(B, "B"), stream.cuda_stream, ctypes.byref(out))
    _check(rc)
    return PackedB(out.value, kind, k, n, B.device)


def pack_b_i16(B, stream=None) -> PackedB:
    """Pack an int16 B (k x n) for gemm_i16_packed."""
    import torch
    return _pack("gemmi_pack_b_i16", "i16", B, torch.int16, stream)


def pack_b_i8(B, stream=None) -> PackedB:
    """Pack an int8 B (k x n) for gemm_i8_packed."""
    import torch
    return _pack("gemmi_pack_b_i8", "i8", B, torch.int8, stream)


def pack_b_i4(B, n, stream=None) -> PackedB:
    """Pack an int4 B for gemm_i4_packed: B a uint8 (k, >= ceil(n/2)) tensor in gemm_i4's format."""
    import torch
    return _pack("gemmi_pack_b_i4", "i4", B, torch.uint8, stream, n=n)


def _packed_call(fn_name, kind, A, Bp, C, op_dtype, c_dtype, stream):
    import torch
    if not isinstance(Bp, PackedB) or Bp.kind != kind:
        raise TypeError(f"B must be a PackedB of kind {kind}")
    for t, nm, dt in ((A, "A", op_dtype), (C, "C", c_dtype)):
        if not isinstance(t, torch.Tensor) or not t.is_cuda or t.dtype != dt:
            raise TypeError(f"{nm} must be a CUDA {dt} tensor")
    m, k = A.shape
    if kind == "i4":  # A packed: k comes from the handle
        k = Bp.k if A.shape[1] >= (Bp.k + 1) // 2 else -1
    if k != Bp.k or tuple(C.shape) != (m, Bp.n):
        raise ValueError(f"shape mismatch: A {tuple(A.shape)}, packed B {(Bp.k, Bp.n)}, C {tuple(C.shape)}")
    if stream is None:
        stream = torch.cuda.current_stream(A.device)
    with torch.cuda.device(A.device):
        rc = getattr(lib(), fn_name)(m, A.data_ptr(), _dev_ld(A, "A"), Bp.handle, C.data_ptr(), _dev_ld(C, "C"),
                                     stream.cuda_stream)
    _check(rc)
    return C


def gemm_i16_packed(A, Bp, C, stream=None):
    """C += A @ B with B pre-packed by pack_b_i16 (bit-identical to gemm_i16)."""
    import torch
    return _packed_call("gemm_i16_packed", "i16", A, Bp, C, torch.int16, torch.int64, stream)


def gemm_i8_packed(A, Bp, C, stream=None):
    """C += A @ B with B pre-packed by pack_b_i8 (bit-identical to gemm_i8)."""
    import torch
    return _packed_call("gemm_i8_packed", "i8", A, Bp, C, torch.int8, torch.int32, stream)


def gemm_i4_packed(A, Bp, C, stream=None):
    """C += A @ B with B pre-packed by pack_b_i4 and A packed as for gemm_i4 (bit-identical to gemm_i4)."""
    import torch
    return _packed_call("gemm_i4_packed", "i4", A, Bp, C, torch.uint8, torch.int32, stream)


# ------------------------------------------------------------------ host-buffer entry points
def _host_ld(x, name):
    import numpy as np
    if not isinstance(x, np.ndarray) or x.ndim != 2:
        raise TypeError(f"{name} must be a 2-D numpy array")
    rows, cols = x.shape
    if x.size == 0 or rows == 1:
        return max(cols, 1)
    if (cols > 1 and x.strides[1] != x.itemsize) or x.strides[0] % x.itemsize or x.strides[0] < cols * x.itemsize:
        raise ValueError(f"{name} must be row-major with unit column stride")
    return x.strides[0] // x.itemsize


def _host_call(fn_name, A, B, C, op_dtype, c_dtype):
    import numpy as np
    for x, nm, dt in ((A, "A", op_dtype), (B, "B", op_dtype), (C, "C", c_dtype)):
        if not isinstance(x, np.ndarray) or x.dtype != dt:
            raise TypeError(f"{nm} must be a numpy {np.dtype(dt).name} array")
    if not C.flags.writeable:
        raise ValueError("C must be writeable")
    m, k = A.shape
    k2, n = B.shape
    if k2 != k or C.shape != (m, n):
        raise ValueError(f"shape mismatch: A {A.shape}, B {B.shape}, C {C.shape}")
    rc = getattr(lib(), fn_name)(m, n, k, A.ctypes.data, _host_ld(A, "A"), B.ctypes.data, _host_ld(B, "B"),
                                 C.ctypes.data, _host_ld(C, "C"))
    _check(rc)
    return C


def gemm_i16_host(A, B, C):
    """C += A @ B for numpy (host) arrays; the library stages the copies and waits for the result."""
    import numpy as np
    return _host_call("gemm_i16_host", A, B, C, np.int16, np.int64)


def gemm_i8_host(A, B, C):
    import numpy as np
    return _host_call("gemm_i8_host", A, B, C, np.int8, np.int32)


def gemm_i4_host(A, B, C, k):
    """gemm_i4 on numpy (host) arrays: A uint8 (m, >= ceil(k/2)) and B uint8 (k, >= ceil(n/2)) packed
    as for gemm_i4, C int32 (m, n)."""
    import numpy as np
    for x, nm, dt in ((A, "A", np.uint8), (B, "B", np.uint8), (C, "C", np.int32)):
        if not isinstance(x, np.ndarray) or x.dtype != dt:
            raise TypeError(f"{nm} must be a numpy {np.dtype(dt).name} array")
    if not C.flags.writeable:
        raise ValueError("C must be writeable")
    m, n = C.shape
    k = int(k)
    if A.ndim != 2 or B.ndim != 2 or A.shape[0] != m or B.shape[0] != k or A.shape[1] < (k + 1) // 2 \
            or B.shape[1] < (n + 1) // 2:
        raise ValueError(f"shape mismatch: packed A {A.shape}, packed B {B.shape}, C {C.shape}, k {k}")
    rc = lib().gemm_i4_host(m, n, k, A.ctypes.data, _host_ld(A, "A"), B.ctypes.data, _host_ld(B, "B"),
                            C.ctypes.data, _host_ld(C, "C"))
    _check(rc)
    return C


# ------------------------------------------------------------------ control
def set_stream(stream) -> None:
    """Stream used by the host-buffer entry points (a torch.cuda.Stream, a raw handle, or None)."""
    handle = getattr(stream, "cuda_stream", stream) or 0
    lib().gemmi_set_stream(ctypes.c_void_p(handle))


def device_status() -> int:
    """Synchronises the device; returns and clears its status word (OK or ETIMEOUT)."""
    return int(lib().gemmi_device_status())


def stream_read_probe(B, stream=None) -> None:
    """Reads the int16 device matrix B the way the skinny-M kernel streams it and discards it
    (gemmi_stream_read_probe): the read floor of that kernel, for measurements."""
    import torch
    if B.dtype != torch.int16 or B.dim() != 2 or B.stride(1) != 1 or not B.is_cuda:
        raise TypeError("the read probe takes a 2-D row-major int16 CUDA tensor")
    handle = getattr(stream, "cuda_stream", stream)
    if handle is None:
        handle = torch.cuda.current_stream().cuda_stream
    _check(lib().gemmi_stream_read_probe(B.shape[0], B.shape[1], B.data_ptr(), B.stride(0), ctypes.c_void_p(handle)))


def device_status_stream(stream=None) -> int:
    """Synchronises one stream (a torch.cuda.Stream, a raw cudaStream_t or None for the legacy
    default stream); returns and clears the device's status words (OK or ETIMEOUT)."""
    handle = getattr(stream, "cuda_stream", stream)
    return int(lib().gemmi_device_status_stream(ctypes.c_void_p(handle or 0)))


def device_status_detail() -> int:
    return int(lib().gemmi_device_status_detail())


def set_option(option: int, value: int) -> None:
    _check(lib().gemmi_set_option(option, value))


def get_option(option: int) -> int:
    return int(lib().gemmi_get_option(option))


def release_workspace() -> None:
    _check(lib().gemmi_release_workspace())


def workspace_bytes() -> int:
    return int(lib().gemmi_workspace_bytes())


def selftest_wait_timeout(timeout_us: int = 1000) -> int:
    return int(lib().gemmi_selftest_wait_timeout(timeout_us))


def kernel_timing(enable: bool) -> None:
    """Switch per-kernel CUDA-event timing on/off (resets the sums)."""
    _check(lib().gemmi_kernel_timing(1 if enable else 0))


def kernel_time(kernel: int):
    """(total milliseconds, launches) of one kernel since timing was switched on."""
    ms, n = ctypes.c_double(0.0), ctypes.c_int64(0)
    _check(lib().gemmi_kernel_time(kernel, ctypes.byref(ms), ctypes.byref(n)))
    return ms.value, n.value


def version() -> str:
    return lib().gemmi_version().decode()
