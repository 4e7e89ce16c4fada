"""Thin ctypes binding over libpifa.so (include/pifa.h). Argument marshalling only: every step of
the forward pass runs in the library's CUDA kernels; the host compression runs in its C++ code.

Functions keep the C names. Tensors are torch tensors (device memory and streams come from
PyTorch); host arrays for pifa_compress are numpy. The library is loaded on first use and a
missing or unloadable library raises -- there is no fallback path.
"""
from __future__ import annotations

import ctypes
import os
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libpifa.so")

PIFA_OK = 0
PIFA_ERR_INVALID_ARG = -1
PIFA_ERR_ALIGNMENT = -2
PIFA_ERR_UNSUPPORTED = -3
PIFA_ERR_CUDA = -4
PIFA_ERR_TIMEOUT = -5
PIFA_ERR_RANK_DEFICIENT = -6
PIFA_ERR_WORKSPACE = -7
PIFA_ERR_DEVICE_INDEX = -8
PIFA_ERR_RANGE = -9

PIFA_DTYPE_BF16 = 0
PIFA_DTYPE_FP16 = 1

PIFA_VARIANT_AUTO = 0
PIFA_VARIANT_DECODE = 1
PIFA_VARIANT_PREFILL_SPLIT = 2
PIFA_VARIANT_PREFILL_FUSED = 3

PIFA_DECODE_GRID_AUTO = 0
PIFA_DECODE_GRID_WAVES = 1
PIFA_DECODE_GRID_PERSISTENT = 2
PIFA_DECODE_GRID_SPLITK = 3

# every symbol include/pifa.h declares
EXPORTS = (
    "pifa_forward", "pifa_forward_variant", "pifa_workspace_size", "pifa_select_variant",
    "pifa_variant_name", "pifa_compress", "pifa_validate_indices", "pifa_device_status",
    "pifa_status_string", "pifa_last_error", "pifa_version", "pifa_forward_decode_noalloc",
    "pifa_set_wait_timeout", "pifa_selftest_wait_timeout", "pifa_launch_count", "pifa_set_decode_grid",
    "pifa_forward_grouped",
    "pifa_workspace_size_grouped", "pifa_compress_device", "pifa_compress_device_workspace_size",
    "pifa_backward", "pifa_backward_workspace_size", "pifa_m_accumulate", "pifa_m_accumulate_workspace_size",
    "pifa_m_reconstruct", "pifa_m_reconstruct_workspace_size",
)


class PifaError(RuntimeError):
    def __init__(self, status: int, where: str, detail: str = ""):
        self.status = status
        name = pifa_status_string(status) if _lib_handle is not None else str(status)
        super().__init__(f"{where}: {name} ({status}) {detail}".rstrip())


class PifaCompressInfo(ctypes.Structure):
    _fields_ = [("min_pivot_gap", ctypes.c_double), ("r_ratio", ctypes.c_double),
                ("max_abs_c", ctypes.c_double), ("threads", ctypes.c_int32)]


_lib_handle = None
_lock = threading.Lock()
_I64 = ctypes.c_int64
_VP = ctypes.c_void_p


def load(path: str | None = None) -> ctypes.CDLL:
    """Load libpifa.so (once) and declare its prototypes. Raises OSError if it cannot load."""
    global _lib_handle
    with _lock:
        if _lib_handle is not None:
            return _lib_handle
        p = path or LIB_PATH
        if not os.path.exists(p):
            raise OSError(f"{p} not found: build it with `python -m paper_2501_19090_gb300.build`")
        lib = ctypes.CDLL(p)
        fwd = [_VP, _I64, _I64, _I64, _VP, _I64, _I64, _VP, _I64, _I64]
        tail = [_VP, _VP, _VP, _I64, _VP, _I64]
        lib.pifa_forward.argtypes = fwd + [ctypes.c_int] + tail + [_VP]
        lib.pifa_forward.restype = ctypes.c_int
        lib.pifa_forward_variant.argtypes = fwd + [ctypes.c_int] + tail + [ctypes.c_int, _VP]
        lib.pifa_forward_variant.restype = ctypes.c_int
        lib.pifa_forward_decode_noalloc.argtypes = fwd + tail[:4] + [_VP]
        lib.pifa_forward_decode_noalloc.restype = ctypes.c_int
        lib.pifa_workspace_size.argtypes = [_I64, _I64, _I64, _I64, ctypes.c_int, ctypes.c_int]
        lib.pifa_workspace_size.restype = _I64
        lib.pifa_forward_grouped.argtypes = [_I64] + fwd + [ctypes.c_int] + tail + [_VP]
        lib.pifa_forward_grouped.restype = ctypes.c_int
        lib.pifa_workspace_size_grouped.argtypes = [_I64, _I64, _I64, _I64, _I64, ctypes.c_int]
        lib.pifa_workspace_size_grouped.restype = _I64
        lib.pifa_select_variant.argtypes = [_I64, _I64, _I64, _I64, ctypes.c_int]
        lib.pifa_select_variant.restype = ctypes.c_int
        lib.pifa_variant_name.argtypes = [ctypes.c_int]
        lib.pifa_variant_name.restype = ctypes.c_char_p
        lib.pifa_compress.argtypes = [_VP, _VP, _I64, _I64, _I64, _VP, _VP, _VP, _I64, _VP, _I64,
                                      ctypes.POINTER(PifaCompressInfo)]
        lib.pifa_compress.restype = ctypes.c_int
        lib.pifa_compress_device.argtypes = [_VP, _VP, _I64, _I64, _I64, _VP, _VP, _VP, _I64, _VP, _I64, _VP, _I64,
                                             ctypes.POINTER(PifaCompressInfo), _VP]
        lib.pifa_compress_device.restype = ctypes.c_int
        lib.pifa_compress_device_workspace_size.argtypes = [_I64, _I64, _I64]
        lib.pifa_compress_device_workspace_size.restype = _I64
        lib.pifa_backward.argtypes = [_VP, _I64, _I64, _I64, _VP, _I64, _I64, _VP, _I64, _I64, _VP, _VP, _VP, _I64,
                                      _VP, _I64, _VP, _I64, _VP, _I64, _VP, _I64, _VP]
        lib.pifa_backward.restype = ctypes.c_int
        lib.pifa_backward_workspace_size.argtypes = [_I64, _I64, _I64, _I64]
        lib.pifa_backward_workspace_size.restype = _I64
        lib.pifa_m_accumulate.argtypes = [_VP, _VP, _I64, _I64, _I64, _VP, _I64, _I64, ctypes.c_float, _VP, _I64,
                                          _VP, _I64, _VP, _I64, _VP]
        lib.pifa_m_accumulate.restype = ctypes.c_int
        lib.pifa_m_accumulate_workspace_size.argtypes = [_I64, _I64, _I64]
        lib.pifa_m_accumulate_workspace_size.restype = _I64
        lib.pifa_m_reconstruct.argtypes = [_VP, _I64, _VP, _I64, _VP, _VP, _I64, _I64, _I64, _I64, ctypes.c_double,
                                           _VP, _VP, _VP, _I64, _VP]
        lib.pifa_m_reconstruct.restype = ctypes.c_int
        lib.pifa_m_reconstruct_workspace_size.argtypes = [_I64, _I64, _I64]
        lib.pifa_m_reconstruct_workspace_size.restype = _I64
        lib.pifa_validate_indices.argtypes = [_VP, _VP, _I64, _I64]
        lib.pifa_validate_indices.restype = ctypes.c_int
        lib.pifa_device_status.argtypes = [_VP]
        lib.pifa_device_status.restype = ctypes.c_int
        lib.pifa_status_string.argtypes = [ctypes.c_int]
        lib.pifa_status_string.restype = ctypes.c_char_p
        lib.pifa_last_error.argtypes = []
        lib.pifa_last_error.restype = ctypes.c_char_p
        lib.pifa_set_wait_timeout.argtypes = [_I64]
        lib.pifa_set_wait_timeout.restype = ctypes.c_int
        lib.pifa_selftest_wait_timeout.argtypes = [_VP]
        lib.pifa_selftest_wait_timeout.restype = ctypes.c_int
        lib.pifa_launch_count.argtypes = []
        lib.pifa_launch_count.restype = ctypes.c_int64
        lib.pifa_set_decode_grid.argtypes = [ctypes.c_int]
        lib.pifa_set_decode_grid.restype = ctypes.c_int
        lib.pifa_version.argtypes = []
        lib.pifa_version.restype = ctypes.c_char_p
        _lib_handle = lib
        return lib


def _lib() -> ctypes.CDLL:
    return _lib_handle if _lib_handle is not None else load()


def _check(status: int, where: str) -> int:
    if status != PIFA_OK:
        raise PifaError(status, where, _lib().pifa_last_error().decode())
    return status


# ---- plain wrappers ------------------------------------------------------------------------------
def pifa_version() -> str:
    return _lib().pifa_version().decode()


def pifa_status_string(status: int) -> str:
    return _lib().pifa_status_string(int(status)).decode()


def pifa_set_wait_timeout(ns: int) -> None:
    """Bound of every device-side wait of later launches, in ns (0 restores the default 1 s)."""
    _check(_lib().pifa_set_wait_timeout(int(ns)), "pifa_set_wait_timeout")


def pifa_set_decode_grid(mode: int) -> None:
    """Layout of the decode phases for later calls: PIFA_DECODE_GRID_AUTO, _WAVES or _PERSISTENT."""
    _check(_lib().pifa_set_decode_grid(int(mode)), "pifa_set_decode_grid")


def pifa_selftest_wait_timeout(stream=None) -> None:
    """Enqueue the bounded-wait self-test kernel (latches PIFA_ERR_TIMEOUT; see include/pifa.h)."""
    _check(_lib().pifa_selftest_wait_timeout(_stream_ptr(stream)), "pifa_selftest_wait_timeout")


def pifa_launch_count() -> int:
    """Kernels the library has enqueued since it was loaded (see include/pifa.h)."""
    return int(_lib().pifa_launch_count())


def pifa_last_error() -> str:
    return _lib().pifa_last_error().decode()


def pifa_variant_name(variant: int) -> str:
    return _lib().pifa_variant_name(int(variant)).decode()


def pifa_select_variant(T: int, m: int, n: int, r: int, c_dtype: int = PIFA_DTYPE_BF16) -> int:
    v = _lib().pifa_select_variant(T, m, n, r, c_dtype)
    if v < 0:
        _check(v, "pifa_select_variant")
    return v


def pifa_workspace_size(T: int, m: int, n: int, r: int, variant: int = PIFA_VARIANT_AUTO,
                        c_dtype: int = PIFA_DTYPE_BF16) -> int:
    v = _lib().pifa_workspace_size(T, m, n, r, c_dtype, variant)
    if v < 0:
        _check(int(v), "pifa_workspace_size")
    return int(v)


def pifa_validate_indices(pivot_idx: np.ndarray, nonpivot_idx: np.ndarray, m: int, r: int) -> int:
    """Host check of the index sets; returns the pifa_status (does not raise)."""
    p = np.ascontiguousarray(pivot_idx, dtype=np.int32)
    q = np.ascontiguousarray(nonpivot_idx, dtype=np.int32)
    return _lib().pifa_validate_indices(p.ctypes.data, q.ctypes.data if q.size else None, m, r)


def pifa_device_status(stream=None) -> int:
    """Synchronize the stream, then read and clear the device error word (a pifa_status)."""
    return _lib().pifa_device_status(_stream_ptr(stream))


def pifa_compress(U: np.ndarray, V: np.ndarray, r: int):
    """Algorithm 1 on the host in float64 (library C++ route). Returns (I, I^c, W_p, C, info)."""
    U = np.ascontiguousarray(U, dtype=np.float64)
    V = np.ascontiguousarray(V, dtype=np.float64)
    m, n = U.shape[0], V.shape[0]
    if U.shape[1] != r or V.shape[1] != r:
        raise ValueError("U must be m x r and V n x r")
    piv = np.empty(r, dtype=np.int32)
    nonpiv = np.empty(m - r, dtype=np.int32)
    Wp = np.empty((r, n), dtype=np.float64)
    C = np.empty((m - r, r), dtype=np.float64)
    info = PifaCompressInfo()
    st = _lib().pifa_compress(U.ctypes.data, V.ctypes.data, m, n, r, piv.ctypes.data,
                              nonpiv.ctypes.data if m > r else None, Wp.ctypes.data, n,
                              C.ctypes.data if m > r else None, r, ctypes.byref(info))
    _check(st, "pifa_compress")
    return piv, nonpiv, Wp, C, info


def pifa_compress_device_workspace_size(m: int, n: int, r: int) -> int:
    v = _lib().pifa_compress_device_workspace_size(m, n, r)
    if v < 0:
        _check(int(v), "pifa_compress_device_workspace_size")
    return int(v)


def pifa_compress_device(U, V, stream=None):
    """Algorithm 1 on the GPU in float64 (pifa_compress_device). U (m x r) and V (n x r) are CUDA
    tensors (converted to contiguous float64 on their device). Returns (I, I^c, W_p, C, info) as
    CUDA tensors (int32, int32, float64, float64) and the host info struct."""
    import torch
    if not (isinstance(U, torch.Tensor) and isinstance(V, torch.Tensor)) or U.device.type != "cuda" or V.device != U.device:
        raise ValueError("pifa: U and V must be CUDA tensors on one device")
    if U.dim() != 2 or V.dim() != 2 or U.shape[1] != V.shape[1]:
        raise ValueError("pifa: U must be m x r and V n x r")
    U = U.to(torch.float64).contiguous()
    V = V.to(torch.float64).contiguous()
    (m, r), n = U.shape, V.shape[0]
    dev = U.device
    need = pifa_compress_device_workspace_size(m, n, r)
    ws = torch.empty(need + 256, dtype=torch.uint8, device=dev)
    ws_ptr = ws.data_ptr() + (-ws.data_ptr()) % 256
    piv = torch.empty(r, dtype=torch.int32, device=dev)
    nonpiv = torch.empty(max(m - r, 1), dtype=torch.int32, device=dev)
    Wp = torch.empty((r, n), dtype=torch.float64, device=dev)
    C = torch.empty((max(m - r, 1), r), dtype=torch.float64, device=dev)
    info = PifaCompressInfo()
    st = _lib().pifa_compress_device(U.data_ptr(), V.data_ptr(), m, n, r, piv.data_ptr(),
                                     nonpiv.data_ptr() if m > r else None, Wp.data_ptr(), n,
                                     C.data_ptr() if m > r else None, r, ws_ptr, need, ctypes.byref(info),
                                     _stream_ptr(stream))
    _check(st, "pifa_compress_device")
    return piv, nonpiv[:m - r], Wp, C[:m - r], info


# ---- forward -------------------------------------------------------------------------------------
def _stream_ptr(stream):
    if stream is None:
        import torch
        if not torch.cuda.is_available():
            return None
        return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, int):
        return ctypes.c_void_p(stream)
    return ctypes.c_void_p(stream.cuda_stream)


_workspaces: dict = {}


def workspace(nbytes: int, device, stream=None, tag: str = ""):
    """A cached device scratch tensor of at least nbytes on `device` (grown, never shrunk).

    The cache is keyed by device, stream and `tag`, so calls on different streams never share
    scratch, and a caller that keeps several calls' scratch apart on one stream tags them.
    """
    import torch
    key = (str(device), 0 if stream is None else getattr(stream, "cuda_stream", stream), str(tag))
    buf = _workspaces.get(key)
    if buf is None or buf.numel() < nbytes:
        buf = torch.empty(max(nbytes, 256) + 256, dtype=torch.uint8, device=device)
        _workspaces[key] = buf
    return buf


def _ld(t) -> int:
    if t.dim() != 2 or t.stride(1) != 1:
        raise ValueError("expected a row-major 2-D tensor with unit column stride")
    return t.stride(0)


def c_dtype_of(C) -> int:
    """The pifa_dtype of a torch tensor C (bfloat16 or float16)."""
    import torch
    if C is None or C.dtype == torch.bfloat16:
        return PIFA_DTYPE_BF16
    if C.dtype == torch.float16:
        return PIFA_DTYPE_FP16
    raise TypeError(f"C must be bfloat16 or float16, got {C.dtype}")


def _operands(G: int, X, Wp, C, pivot_idx, nonpivot_idx, Y, workspace_tensor=None, c_fp16_ok=True):
    """Check what the C ABI cannot see -- tensor type, dtype, shape and device -- before any
    pointer reaches the library (a host or mistyped buffer would otherwise be read as device
    bf16). Types and shapes first, then that every tensor sits on X's CUDA device. Returns
    (T, n, r, m) of one group. Raises ValueError."""
    import torch

    def fail(msg):
        raise ValueError(f"pifa: {msg}")

    def tensor(name, t):
        if not isinstance(t, torch.Tensor):
            fail(f"{name} must be a torch tensor")
        return t

    if tensor("X", X).dim() != 2 or X.dtype != torch.bfloat16:
        fail(f"X must be a 2-D bfloat16 tensor (T x n) (it is {X.dtype} {tuple(X.shape)})")
    T, n = X.shape
    if tensor("Wp", Wp).dim() != 2 or Wp.dtype != torch.bfloat16 or Wp.shape[1] != n or Wp.shape[0] % G:
        fail(f"Wp must be a bfloat16 ({G} r) x {n} tensor (it is {Wp.dtype} {tuple(Wp.shape)})")
    r = Wp.shape[0] // G
    for name, t in (("pivot_idx", pivot_idx), ("nonpivot_idx", nonpivot_idx)):
        if t is not None and (tensor(name, t).dim() != 1 or t.dtype != torch.int32 or not t.is_contiguous()):
            fail(f"{name} must be a contiguous 1-D int32 tensor (it is {t.dtype} {tuple(t.shape)})")
    if pivot_idx is None or pivot_idx.numel() != G * r:
        fail(f"pivot_idx must hold {G * r} indices")
    nnp = nonpivot_idx.numel() if nonpivot_idx is not None else 0
    if nnp % G:
        fail("nonpivot_idx must hold the same number of indices for every group")
    m = r + nnp // G
    if m > r:
        ok = (torch.bfloat16, torch.float16) if c_fp16_ok else (torch.bfloat16,)
        if tensor("C", C).dim() != 2 or C.dtype not in ok or tuple(C.shape) != (G * (m - r), r):
            fail(f"C must be a {'bfloat16 or float16' if c_fp16_ok else 'bfloat16'} tensor of shape "
                 f"{(G * (m - r), r)} (it is {C.dtype} {tuple(C.shape)})")
    if Y is not None and (tensor("Y", Y).dim() != 2 or Y.dtype != torch.bfloat16 or tuple(Y.shape) != (T, G * m)):
        fail(f"Y must be a bfloat16 tensor of shape {(T, G * m)} (it is {Y.dtype} {tuple(Y.shape)})")
    if workspace_tensor is not None:
        tensor("workspace_tensor", workspace_tensor)
    dev = X.device
    if dev.type != "cuda":
        fail(f"X must be a CUDA tensor (it is on {dev})")
    for name, t in (("Wp", Wp), ("C", C if m > r else None), ("pivot_idx", pivot_idx),
                    ("nonpivot_idx", nonpivot_idx), ("Y", Y), ("workspace_tensor", workspace_tensor)):
        if t is not None and t.device != dev:
            fail(f"{name} is on {t.device}, X on {dev}")
    return T, n, r, m


def pifa_forward(X, Wp, C, pivot_idx, nonpivot_idx, Y=None, variant: int = PIFA_VARIANT_AUTO,
                 workspace_tensor=None, stream=None):
    """Y = PIFA(X) through pifa_forward_variant. X (T x n), Wp (r x n) bf16 CUDA tensors; C
    ((m-r) x r) bf16 or fp16; pivot_idx / nonpivot_idx int32 CUDA tensors. Allocates Y (T x m)
    if not given."""
    import torch
    T, n, r, m = _operands(1, X, Wp, C, pivot_idx, nonpivot_idx, Y, workspace_tensor)
    if Y is None:
        Y = torch.empty((T, m), dtype=torch.bfloat16, device=X.device)
    has_np = m > r
    cdt = c_dtype_of(C if has_np else None)
    need = pifa_workspace_size(T, m, n, r, variant, cdt)
    ws = workspace_tensor
    if need > 0 and ws is None:
        ws = workspace(need, X.device, stream)
    ws_ptr = 0 if ws is None else ws.data_ptr()
    if ws is not None and ws_ptr % 256:
        ws_ptr += 256 - ws_ptr % 256
    ws_bytes = 0 if ws is None else ws.numel() * ws.element_size() - (ws_ptr - ws.data_ptr())
    st = _lib().pifa_forward_variant(
        X.data_ptr(), T, n, _ld(X), Wp.data_ptr(), r, _ld(Wp),
        C.data_ptr() if has_np else None, m, _ld(C) if has_np else r, cdt,
        pivot_idx.data_ptr(), nonpivot_idx.data_ptr() if has_np else None,
        Y.data_ptr(), _ld(Y), ws_ptr or None, ws_bytes, variant, _stream_ptr(stream))
    _check(st, "pifa_forward")
    return Y


def pifa_workspace_size_grouped(groups: int, T: int, m: int, n: int, r: int, c_dtype: int = PIFA_DTYPE_BF16) -> int:
    v = _lib().pifa_workspace_size_grouped(groups, T, m, n, r, c_dtype)
    if v < 0:
        _check(int(v), "pifa_workspace_size_grouped")
    return int(v)


def pifa_forward_grouped(groups: int, X, Wp, C, pivot_idx, nonpivot_idx, Y=None, workspace_tensor=None, stream=None):
    """Y = [PIFA_0(X) | ... | PIFA_{G-1}(X)] for G layers of one shape sharing X, through
    pifa_forward_grouped: Wp (G r x n) and C (G (m-r) x r) hold the groups' matrices stacked by
    rows; pivot_idx / nonpivot_idx the groups' indices offset by g m. Allocates Y (T x G m) if not
    given."""
    import torch
    G = int(groups)
    if G < 1:
        raise ValueError("pifa: groups must be >= 1")
    T, n, r, m = _operands(G, X, Wp, C, pivot_idx, nonpivot_idx, Y, workspace_tensor)
    if Y is None:
        Y = torch.empty((T, G * m), dtype=torch.bfloat16, device=X.device)
    cdt = c_dtype_of(C)
    need = pifa_workspace_size_grouped(G, T, m, n, r, cdt)
    ws = workspace_tensor
    if need > 0 and ws is None:
        ws = workspace(need, X.device, stream)
    ws_ptr = 0 if ws is None else ws.data_ptr()
    if ws is not None and ws_ptr % 256:
        ws_ptr += 256 - ws_ptr % 256
    ws_bytes = 0 if ws is None else ws.numel() * ws.element_size() - (ws_ptr - ws.data_ptr())
    st = _lib().pifa_forward_grouped(
        G, X.data_ptr(), T, n, _ld(X), Wp.data_ptr(), r, _ld(Wp), C.data_ptr(), m, _ld(C), cdt,
        pivot_idx.data_ptr(), nonpivot_idx.data_ptr(), Y.data_ptr(), _ld(Y), ws_ptr or None, ws_bytes,
        _stream_ptr(stream))
    _check(st, "pifa_forward_grouped")
    return Y


def pifa_forward_decode_noalloc(X, Wp, C, pivot_idx, nonpivot_idx, Y=None, stream=None):
    """Decode forward (T <= 16) without a workspace: the library's static 1 MiB device scratch
    is used instead (see include/pifa.h). Allocates Y here only if the caller passes none."""
    import torch
    T, n, r, m = _operands(1, X, Wp, C, pivot_idx, nonpivot_idx, Y, c_fp16_ok=False)
    if Y is None:
        Y = torch.empty((T, m), dtype=torch.bfloat16, device=X.device)
    has_np = m > r
    st = _lib().pifa_forward_decode_noalloc(
        X.data_ptr(), T, n, _ld(X), Wp.data_ptr(), r, _ld(Wp),
        C.data_ptr() if has_np else None, m, _ld(C) if has_np else r,
        pivot_idx.data_ptr(), nonpivot_idx.data_ptr() if has_np else None,
        Y.data_ptr(), _ld(Y), _stream_ptr(stream))
    _check(st, "pifa_forward_decode_noalloc")
    return Y


def pifa_backward_workspace_size(T: int, m: int, n: int, r: int) -> int:
    v = int(_lib().pifa_backward_workspace_size(T, m, n, r))
    if v < 0:
        _check(v, "pifa_backward_workspace_size")
    return v


def pifa_m_accumulate_workspace_size(T: int, m: int, n: int) -> int:
    v = int(_lib().pifa_m_accumulate_workspace_size(T, m, n))
    if v < 0:
        _check(v, "pifa_m_accumulate_workspace_size")
    return v


def pifa_backward(X, Wp, C, pivot_idx, nonpivot_idx, dY, want=("dX", "dWp", "dC"), workspace_tensor=None,
                  stream=None):
    """Gradients of the forward pass through pifa_backward: returns (dX bf16 T x n, dW_p fp32 r x n,
    dC fp32 (m-r) x r), each None unless named in `want`. Tensors as pifa_forward (C bf16); dY is
    a bf16 CUDA tensor T x m."""
    import torch
    T, n, r, m = _operands(1, X, Wp, C, pivot_idx, nonpivot_idx, None, workspace_tensor, c_fp16_ok=False)
    if not isinstance(dY, torch.Tensor) or dY.dtype != torch.bfloat16 or tuple(dY.shape) != (T, m) or dY.device != X.device:
        raise ValueError(f"pifa: dY must be a bfloat16 tensor of shape {(T, m)} on {X.device}")
    dev = X.device
    has_np = m > r
    def out(rows, cols, dtype, per16):  # row pitch a multiple of 16 bytes; returns the rows x cols view
        ld = (cols + per16 - 1) // per16 * per16
        return torch.empty((rows, ld), dtype=dtype, device=dev)[:, :cols]

    dX = out(T, n, torch.bfloat16, 8) if "dX" in want else None
    dWp = out(r, n, torch.float32, 4) if "dWp" in want else None
    dC = out(m - r, r, torch.float32, 4) if ("dC" in want and has_np) else None
    need = pifa_backward_workspace_size(T, m, n, r)
    ws = workspace_tensor if workspace_tensor is not None else workspace(need, dev, stream, tag="backward")
    ws_ptr = ws.data_ptr() + (-ws.data_ptr()) % 256
    ws_bytes = ws.numel() * ws.element_size() - (ws_ptr - ws.data_ptr())
    st = _lib().pifa_backward(
        X.data_ptr(), T, n, _ld(X), Wp.data_ptr(), r, _ld(Wp), C.data_ptr() if has_np else None, m,
        _ld(C) if has_np else r, pivot_idx.data_ptr(), nonpivot_idx.data_ptr() if has_np else None,
        dY.data_ptr(), _ld(dY), dX.data_ptr() if dX is not None else None, _ld(dX) if dX is not None else n,
        dWp.data_ptr() if dWp is not None else None, _ld(dWp) if dWp is not None else n,
        dC.data_ptr() if dC is not None else None, _ld(dC) if dC is not None else r,
        ws_ptr, ws_bytes, _stream_ptr(stream))
    _check(st, "pifa_backward")
    return dX, dWp, dC


def pifa_m_accumulate(Xo, Xu, W, lam, XXt, YtXt=None, workspace_tensor=None, stream=None):
    """One calibration batch into the M accumulators (pifa_m_accumulate): XXt (fp32 n x n, its
    upper triangle: X X^T is symmetric) and YtXt (fp32 m x n, optional) are updated in place.
    Xo, Xu bf16 T x n; W bf16 m x n."""
    import torch
    for name, t in (("Xu", Xu), ("XXt", XXt)):
        if not isinstance(t, torch.Tensor) or t.device.type != "cuda":
            raise ValueError(f"pifa: {name} must be a CUDA tensor")
    if Xu.dtype != torch.bfloat16 or Xu.dim() != 2:
        raise ValueError("pifa: Xu must be a 2-D bfloat16 tensor")
    T, n = Xu.shape
    if XXt.dtype != torch.float32 or tuple(XXt.shape) != (n, n):
        raise ValueError(f"pifa: XXt must be a float32 tensor of shape {(n, n)}")
    m = 1
    if YtXt is not None:
        if Xo is None or W is None or Xo.dtype != torch.bfloat16 or tuple(Xo.shape) != (T, n) or _ld(Xo) != _ld(Xu):
            raise ValueError("pifa: Xo must be a bfloat16 tensor shaped and strided like Xu")
        if W.dtype != torch.bfloat16 or W.dim() != 2 or W.shape[1] != n:
            raise ValueError("pifa: W must be a bfloat16 m x n tensor")
        m = W.shape[0]
        if YtXt.dtype != torch.float32 or tuple(YtXt.shape) != (m, n):
            raise ValueError(f"pifa: YtXt must be a float32 tensor of shape {(m, n)}")
        for name, t in (("Xo", Xo), ("W", W), ("YtXt", YtXt)):
            if t.device != Xu.device:
                raise ValueError(f"pifa: {name} is on {t.device}, Xu on {Xu.device}")
    if XXt.device != Xu.device:
        raise ValueError("pifa: XXt must be on Xu's device")
    need = pifa_m_accumulate_workspace_size(T, m, n)
    ws = workspace_tensor if workspace_tensor is not None else workspace(need, Xu.device, stream, tag="macc")
    ws_ptr = ws.data_ptr() + (-ws.data_ptr()) % 256
    ws_bytes = ws.numel() * ws.element_size() - (ws_ptr - ws.data_ptr())
    st = _lib().pifa_m_accumulate(
        Xo.data_ptr() if YtXt is not None else None, Xu.data_ptr(), T, n, _ld(Xu),
        W.data_ptr() if YtXt is not None else None, m, _ld(W) if YtXt is not None else n, float(lam),
        XXt.data_ptr(), _ld(XXt), YtXt.data_ptr() if YtXt is not None else None,
        _ld(YtXt) if YtXt is not None else n, ws_ptr, ws_bytes, _stream_ptr(stream))
    _check(st, "pifa_m_accumulate")
    return XXt, YtXt


def pifa_m_reconstruct(XXt, YtXt, V, W=None, alpha=0.0, stream=None):
    """The M reconstruction (pifa_m_reconstruct): U_r (Eq. 4) and V_r (Eq. 8) in float64 from the
    fp32 accumulators XXt (n x n) and YtXt (m x n), V (n x r, converted to float64) and, for
    alpha > 0, the dense W (bf16 m x n). Returns (U_r, V_r) as float64 CUDA tensors."""
    import torch
    n = XXt.shape[0]
    m = YtXt.shape[0]
    for name, t in (("XXt", XXt), ("YtXt", YtXt)):
        if not isinstance(t, torch.Tensor) or t.dtype != torch.float32 or t.dim() != 2 or t.device.type != "cuda":
            raise ValueError(f"pifa: {name} must be a 2-D float32 CUDA tensor")
    if tuple(XXt.shape) != (n, n) or YtXt.shape[1] != n:
        raise ValueError("pifa: XXt must be n x n and YtXt m x n")
    V = V.to(device=XXt.device, dtype=torch.float64).contiguous()
    if V.dim() != 2 or V.shape[0] != n:
        raise ValueError("pifa: V must be n x r")
    r = V.shape[1]
    if alpha and (W is None or W.dtype != torch.bfloat16 or tuple(W.shape) != (m, n)):
        raise ValueError("pifa: alpha > 0 needs W, a bfloat16 m x n tensor")
    need = int(_lib().pifa_m_reconstruct_workspace_size(m, n, r))
    if need < 0:
        _check(need, "pifa_m_reconstruct_workspace_size")
    ws = torch.empty(need + 256, dtype=torch.uint8, device=XXt.device)
    ws_ptr = ws.data_ptr() + (-ws.data_ptr()) % 256
    U_r = torch.empty((m, r), dtype=torch.float64, device=XXt.device)
    V_r = torch.empty((n, r), dtype=torch.float64, device=XXt.device)
    st = _lib().pifa_m_reconstruct(XXt.data_ptr(), _ld(XXt), YtXt.data_ptr(), _ld(YtXt), V.data_ptr(),
                                   W.data_ptr() if (alpha and W is not None) else None, _ld(W) if (alpha and W is not None) else n,
                                   m, n, r, float(alpha), U_r.data_ptr(), V_r.data_ptr(), ws_ptr, need,
                                   _stream_ptr(stream))
    _check(st, "pifa_m_reconstruct")
    return U_r, V_r
