"""ctypes binding of libgrkv.so: the C ABI of include/grkv.h, same names.

Argument marshalling only: torch tensors are passed as device pointers, the
torch stream as a cudaStream_t.  Every step of the path runs in the CUDA
library; there is no fallback, and `load()` raises if the library is absent.
"""
from __future__ import annotations

import ctypes
import math
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libgrkv.so")

GRKV_OK = 0
GRKV_ERR_INVALID_ARG = -1
GRKV_ERR_UNSUPPORTED = -2
GRKV_ERR_WORKSPACE_TOO_SMALL = -3
GRKV_ERR_MISALIGNED = -4
GRKV_ERR_CUDA = -5
GRKV_ERR_NUMERIC = -6
GRKV_ERR_TIMEOUT = -7
GRKV_ERR_BOUNDS = -8

GRKV_F32 = 0
GRKV_BF16 = 1
GRKV_POOL_MAX = 0
GRKV_POOL_AVG = 1
GRKV_UPDATE_K = 0x1
GRKV_FORCE_SIMT = 0x2
GRKV_ONE_READ_SCORE = 0x4
GRKV_DETERMINISTIC = 0x8
GRKV_CHECKS = 0x10
GRKV_TEST_TIMEOUT = 0x80000000

EXPORTS = ("grkv_params_init", "grkv_workspace_size", "grkv_score", "grkv_select", "grkv_merge",
           "grkv_compress", "grkv_status", "grkv_strerror", "grkv_launch_count",
           "grkv_select_noalloc", "grkv_transfer_workspace_size", "grkv_transfer_check",
           "grkv_compress_ragged_workspace_size", "grkv_compress_ragged")


class grkv_params(ctypes.Structure):
    _fields_ = [
        ("units", ctypes.c_int32), ("group", ctypes.c_int32), ("n", ctypes.c_int32),
        ("d", ctypes.c_int32), ("window", ctypes.c_int32), ("budget", ctypes.c_int32),
        ("pool_kernel", ctypes.c_int32), ("pool_type", ctypes.c_int32),
        ("n_sink", ctypes.c_int32), ("beta", ctypes.c_float), ("lambda_v", ctypes.c_float),
        ("lambda_k", ctypes.c_float), ("scale", ctypes.c_float), ("causal", ctypes.c_int32),
        ("dtype", ctypes.c_int32), ("flags", ctypes.c_uint32), ("cg_iters", ctypes.c_int32),
        ("cg_tol", ctypes.c_float), ("steps", ctypes.c_int32), ("step_tol", ctypes.c_float),
    ]


class GrkvError(RuntimeError):
    def __init__(self, code: int, what: str):
        super().__init__(f"{what}: {strerror(code)} ({code})")
        self.code = code


_lib = None
_P = ctypes.POINTER(grkv_params)
_vp = ctypes.c_void_p


def load():
    """Load the in-tree library (built by paper_2605_31105_gb300.build)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: run __graft_entry__.build() first")
    lib = ctypes.CDLL(LIB_PATH)
    lib.grkv_params_init.argtypes = [_P, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
                                     ctypes.c_int32, ctypes.c_int32]
    lib.grkv_params_init.restype = None
    lib.grkv_workspace_size.argtypes = [_P, ctypes.POINTER(ctypes.c_size_t)]
    lib.grkv_score.argtypes = [_P, _vp, _vp, _vp, _vp, _vp, _vp, _vp, ctypes.c_size_t, _vp]
    lib.grkv_select.argtypes = [_P, _vp, _vp, _vp, ctypes.c_size_t, _vp]
    lib.grkv_merge.argtypes = [_P, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp,
                               ctypes.c_size_t, _vp]
    lib.grkv_compress.argtypes = [_P, _vp, _vp, _vp, _vp, _vp, _vp, _vp, ctypes.c_size_t, _vp]
    lib.grkv_status.argtypes = [_vp, ctypes.POINTER(ctypes.c_int), _vp]
    lib.grkv_strerror.argtypes = [ctypes.c_int]
    lib.grkv_strerror.restype = ctypes.c_char_p
    lib.grkv_select_noalloc.argtypes = [_P, _vp, _vp, _vp]
    lib.grkv_select_noalloc.restype = ctypes.c_int
    lib.grkv_launch_count.argtypes = []
    lib.grkv_launch_count.restype = ctypes.c_uint64
    lib.grkv_transfer_workspace_size.argtypes = [_P, ctypes.c_int32, ctypes.POINTER(ctypes.c_size_t)]
    lib.grkv_transfer_check.argtypes = [_P, ctypes.c_int32, _vp, _vp, _vp, _vp, _vp, _vp, _vp,
                                        _vp, _vp, ctypes.c_size_t, _vp]
    _ip = ctypes.POINTER(ctypes.c_int32)
    lib.grkv_compress_ragged_workspace_size.argtypes = [_P, _ip, ctypes.POINTER(ctypes.c_size_t)]
    lib.grkv_compress_ragged.argtypes = [_P, _ip, _vp, _vp, _vp, _vp, _vp, _vp, _vp,
                                         ctypes.c_size_t, _vp]
    for name in ("grkv_workspace_size", "grkv_score", "grkv_select", "grkv_merge",
                 "grkv_compress", "grkv_status", "grkv_transfer_workspace_size",
                 "grkv_transfer_check", "grkv_compress_ragged_workspace_size",
                 "grkv_compress_ragged"):
        getattr(lib, name).restype = ctypes.c_int
    _lib = lib
    return lib


def strerror(code: int) -> str:
    return load().grkv_strerror(code).decode()


def params(units, group, n, window, budget, **kw) -> grkv_params:
    """grkv_params with the library defaults, then any field overridden by name
    (dtype may be given as "bf16" / "f32")."""
    p = grkv_params()
    load().grkv_params_init(ctypes.byref(p), units, group, n, window, budget)
    for key, val in kw.items():
        if key == "dtype" and isinstance(val, str):
            val = {"bf16": GRKV_BF16, "f32": GRKV_F32}[val]
        if key == "pool_type" and isinstance(val, str):
            val = {"max": GRKV_POOL_MAX, "avg": GRKV_POOL_AVG}[val]
        if key == "lambda_v" and val == math.inf:
            val = float("inf")
        setattr(p, key, val)
    return p


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _check(rc: int, what: str, raise_on_error: bool):
    if rc != GRKV_OK and raise_on_error:
        raise GrkvError(rc, what)
    return rc


def grkv_workspace_size(p: grkv_params) -> int:
    n = ctypes.c_size_t(0)
    _check(load().grkv_workspace_size(ctypes.byref(p), ctypes.byref(n)), "grkv_workspace_size",
           True)
    return n.value


def grkv_score(p, q, k, v, scores, y, row_stats, ws, ws_bytes=None, stream=None, check=True):
    ws_bytes = ws.numel() * ws.element_size() if ws_bytes is None else ws_bytes
    rc = load().grkv_score(ctypes.byref(p), _ptr(q), _ptr(k), _ptr(v), _ptr(scores), _ptr(y),
                           _ptr(row_stats), _ptr(ws), ws_bytes, _stream(stream))
    return _check(rc, "grkv_score", check)


def grkv_select(p, scores, idx, ws, ws_bytes=None, stream=None, check=True):
    ws_bytes = ws.numel() * ws.element_size() if ws_bytes is None else ws_bytes
    rc = load().grkv_select(ctypes.byref(p), _ptr(scores), _ptr(idx), _ptr(ws), ws_bytes,
                            _stream(stream))
    return _check(rc, "grkv_select", check)


def grkv_merge(p, q, k, v, scores, y, idx, k_out, v_out, ws, ws_bytes=None, stream=None,
               check=True, row_stats=None):
    ws_bytes = ws.numel() * ws.element_size() if ws_bytes is None else ws_bytes
    rc = load().grkv_merge(ctypes.byref(p), _ptr(q), _ptr(k), _ptr(v), _ptr(scores), _ptr(y),
                           _ptr(row_stats), _ptr(idx), _ptr(k_out), _ptr(v_out), _ptr(ws),
                           ws_bytes, _stream(stream))
    return _check(rc, "grkv_merge", check)


def grkv_compress(p, q, k, v, k_out, v_out, idx, ws, ws_bytes=None, stream=None, check=True):
    ws_bytes = ws.numel() * ws.element_size() if ws_bytes is None else ws_bytes
    rc = load().grkv_compress(ctypes.byref(p), _ptr(q), _ptr(k), _ptr(v), _ptr(k_out),
                              _ptr(v_out), _ptr(idx), _ptr(ws), ws_bytes, _stream(stream))
    return _check(rc, "grkv_compress", check)


def grkv_select_noalloc(p, scores, idx, stream=None, check=True):
    """grkv_select with the library's built-in scratch array (no workspace)."""
    rc = load().grkv_select_noalloc(ctypes.byref(p), _ptr(scores), _ptr(idx), _stream(stream))
    return _check(rc, "grkv_select_noalloc", check)


def grkv_transfer_workspace_size(p, held: int) -> int:
    n = ctypes.c_size_t(0)
    _check(load().grkv_transfer_workspace_size(ctypes.byref(p), held, ctypes.byref(n)),
           "grkv_transfer_workspace_size", True)
    return n.value


def grkv_transfer_check(p, held, q_win, q_held, k, v, idx, k_out, v_out, report, ws,
                        ws_bytes=None, stream=None, check=True):
    """Decode-side transfer check: report [U][8] fp32 (see include/grkv.h)."""
    ws_bytes = ws.numel() * ws.element_size() if ws_bytes is None else ws_bytes
    rc = load().grkv_transfer_check(ctypes.byref(p), held, _ptr(q_win), _ptr(q_held), _ptr(k),
                                    _ptr(v), _ptr(idx), _ptr(k_out), _ptr(v_out), _ptr(report),
                                    _ptr(ws), ws_bytes, _stream(stream))
    return _check(rc, "grkv_transfer_check", check)


def _budgets(budgets):
    arr = (ctypes.c_int32 * len(budgets))(*[int(x) for x in budgets])
    return arr


def grkv_compress_ragged_workspace_size(p, budgets) -> int:
    n = ctypes.c_size_t(0)
    _check(load().grkv_compress_ragged_workspace_size(ctypes.byref(p), _budgets(budgets),
                                                      ctypes.byref(n)),
           "grkv_compress_ragged_workspace_size", True)
    return n.value


def grkv_compress_ragged(p, budgets, q, k, v, k_out, v_out, idx, ws, ws_bytes=None,
                         stream=None, check=True):
    """grkv_compress with one budget per unit (host list); packed outputs."""
    ws_bytes = ws.numel() * ws.element_size() if ws_bytes is None else ws_bytes
    rc = load().grkv_compress_ragged(ctypes.byref(p), _budgets(budgets), _ptr(q), _ptr(k),
                                     _ptr(v), _ptr(k_out), _ptr(v_out), _ptr(idx), _ptr(ws),
                                     ws_bytes, _stream(stream))
    return _check(rc, "grkv_compress_ragged", check)


def grkv_launch_count() -> int:
    return int(load().grkv_launch_count())


def grkv_status(ws, stream=None) -> int:
    st = ctypes.c_int(0)
    _check(load().grkv_status(_ptr(ws), ctypes.byref(st), _stream(stream)), "grkv_status", True)
    return st.value
