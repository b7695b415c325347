"""Thin ctypes binding of libaio (include/aio.h): same names, argument marshalling only.

Every computation runs in libaio's CUDA kernels.  Device buffers are passed as
integer addresses (e.g. ``tensor.data_ptr()``) and streams as integer handles
(``torch.cuda.current_stream().cuda_stream``).  A non-OK status raises AioError
carrying the code and libaio's detail message.  There is no fallback: if
libaio.so is missing, importing this module raises.
"""
from __future__ import annotations

import ctypes
import os
import re

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libaio.so")
HEADER = os.path.join(os.path.dirname(_HERE), "include", "aio.h")

if not os.path.exists(LIB_PATH):
    raise ImportError(f"{LIB_PATH} is missing: build it with __graft_entry__.build() (nvcc, sm_103a)")

_lib = ctypes.CDLL(LIB_PATH)

# status codes and flags, read from the header so the binding cannot drift from it
_hdr = open(HEADER).read() if os.path.exists(HEADER) else ""
AIO_OK = 0
AIO_ERR_INVALID_ARG = 1
AIO_ERR_UNSUPPORTED = 2
AIO_ERR_ALIGNMENT = 3
AIO_ERR_CUDA = 4
AIO_ERR_OOM = 5
AIO_ERR_STATE = 6
AIO_ERR_DEVICE_TIMEOUT = 7
AIO_W_BF16 = 0
AIO_W_INT8_PERCHANNEL = 1
AIO_FLAG_ROWMAJOR = 0x1
AIO_FLAG_NO_PDL = 0x2
AIO_FLAG_STREAM_KERNEL = 0x4
AIO_FLAG_TEST_STALL = 0x100
AIO_STEP_GRAPH = 0x1
AIO_STEP_PDL = 0x2
AIO_STEP_PERSISTENT = 0x4
AIO_ROWS_PER_GROUP = 16
AIO_K_TILE = 256
AIO_NOALLOC_SCRATCH_BYTES = 1048576
AIO_ABI_VERSION = 8
AIO_X_GIVEN = 0
AIO_X_RMSNORM = 1
AIO_X_SWIGLU = 2
AIO_X_SLICE = 3
AIO_X_ATTENTION = 4
for _name, _val in re.findall(r"#define\s+(AIO_\w+)\s+(0x[0-9a-fA-F]+|\d+)u?\b", _hdr):
    if _name in globals() and globals()[_name] != int(_val, 0):
        raise ImportError(f"binding constant {_name} disagrees with include/aio.h")


class AioError(RuntimeError):
    def __init__(self, status: int, func: str):
        self.status = status
        detail = _lib.aio_last_error().decode(errors="replace")
        name = _lib.aio_status_string(status).decode()
        super().__init__(f"{func}: {name}: {detail}")


class aio_proj(ctypes.Structure):
    _fields_ = [("h", ctypes.c_void_p), ("x", ctypes.c_void_p), ("W", ctypes.c_void_p),
                ("scales", ctypes.c_void_p), ("y", ctypes.c_void_p)]


class aio_xprep(ctypes.Structure):
    _fields_ = [("op", ctypes.c_int), ("src", ctypes.c_void_p), ("src_stride", ctypes.c_int),
                ("src_off", ctypes.c_int), ("h_in", ctypes.c_void_p), ("h_out", ctypes.c_void_p),
                ("gamma", ctypes.c_void_p), ("eps", ctypes.c_float), ("kv_cache", ctypes.c_void_p),
                ("L_past", ctypes.c_void_p), ("n_heads", ctypes.c_int), ("L_max", ctypes.c_int)]


_vp, _int, _u = ctypes.c_void_p, ctypes.c_int, ctypes.c_uint
_sz, _ll = ctypes.c_size_t, ctypes.c_longlong
_SIGS = {
    "aio_abi_version": (_int, []),
    "aio_status_string": (ctypes.c_char_p, [_int]),
    "aio_last_error": (ctypes.c_char_p, []),
    "aio_linear_create": (_int, [ctypes.POINTER(_vp), _int, _int, _int, _int, _u]),
    "aio_linear_packed_bytes": (_int, [_vp, ctypes.POINTER(_sz), ctypes.POINTER(_sz)]),
    "aio_linear_launch_info": (_int, [_vp, ctypes.POINTER(_int), ctypes.POINTER(_int), ctypes.POINTER(_sz),
                                      ctypes.POINTER(_ll)]),
    "aio_linear_pack": (_int, [_vp, _vp, _vp, _vp, _vp, _vp]),
    "aio_linear_unpack": (_int, [_vp, _vp, _vp, _vp]),
    "aio_linear_run": (_int, [_vp, _vp, _int, _int, _int, _vp, _vp, _vp, _vp]),
    "aio_linear_run_noalloc": (_int, [_vp, _int, _int, _int, _int, _u, _vp, _vp, _vp, _vp, _vp]),
    "aio_linear_check": (_int, [_vp, ctypes.POINTER(_int)]),
    "aio_linear_reset": (_int, [_vp]),
    "aio_linear_destroy": (_int, [_vp]),
    "aio_decode_step_create": (_int, [ctypes.POINTER(_vp), ctypes.POINTER(aio_proj), _int, _int, _u]),
    "aio_decode_step_create_chained": (_int, [ctypes.POINTER(_vp), ctypes.POINTER(aio_proj),
                                              ctypes.POINTER(aio_xprep), _int, _int, _u]),
    "aio_decode_step": (_int, [_vp, _vp]),
    "aio_decode_step_host": (_int, [_vp, _vp, _vp, _sz, _vp, _vp, _sz, _vp]),
    "aio_decode_step_kernels": (_int, [_vp, ctypes.POINTER(_int)]),
    "aio_decode_step_check": (_int, [_vp, ctypes.POINTER(_int)]),
    "aio_decode_step_reset": (_int, [_vp]),
    "aio_decode_step_destroy": (_int, [_vp]),
    "aio_probe_read": (_int, [_vp, _sz, _vp, _vp]),
    "aio_attention_workspace_bytes": (_int, [_int, ctypes.POINTER(_sz)]),
    "aio_attention_decode": (_int, [_vp, _int, _vp, _vp, _int, _int, _int, _int, _int, _vp, _vp, _sz, _vp]),
    "aio_attention_check": (_int, [_vp, ctypes.POINTER(_int)]),
    "aio_pld_draft": (_int, [_vp, _int, _int, _int, _vp, _vp]),
    "aio_argmax_rows": (_int, [_vp, _int, _int, _int, _vp, _vp]),
    "aio_pld_accept": (_int, [_vp, _vp, _vp, _vp]),
    "aio_route": (_int, [_vp, _vp, _int, _int, _int, ctypes.c_float, _vp, _vp]),
}
for _f, (_res, _args) in _SIGS.items():
    _fn = getattr(_lib, _f)
    _fn.restype = _res
    _fn.argtypes = _args
if _lib.aio_abi_version() != AIO_ABI_VERSION:
    raise ImportError(f"{LIB_PATH} has ABI version {_lib.aio_abi_version()}, the binding expects "
                      f"{AIO_ABI_VERSION}: rebuild it (paper_2604_09752_gb300.build)")


def lib():
    return _lib


def _check(status: int, func: str):
    if status != AIO_OK:
        raise AioError(status, func)


def aio_abi_version() -> int:
    return _lib.aio_abi_version()


def aio_status_string(s: int) -> str:
    return _lib.aio_status_string(s).decode()


def aio_last_error() -> str:
    return _lib.aio_last_error().decode(errors="replace")


def aio_linear_create(K: int, N: int, wt: int, max_M: int, flags: int = 0) -> int:
    h = _vp()
    _check(_lib.aio_linear_create(ctypes.byref(h), K, N, wt, max_M, flags), "aio_linear_create")
    return h.value


def aio_linear_packed_bytes(h: int):
    w, s = _sz(), _sz()
    _check(_lib.aio_linear_packed_bytes(h, ctypes.byref(w), ctypes.byref(s)), "aio_linear_packed_bytes")
    return w.value, s.value


def aio_linear_launch_info(h: int):
    g, b, sm, t = _int(), _int(), _sz(), _ll()
    _check(_lib.aio_linear_launch_info(h, ctypes.byref(g), ctypes.byref(b), ctypes.byref(sm), ctypes.byref(t)),
           "aio_linear_launch_info")
    return {"grid": g.value, "block": b.value, "smem_bytes": sm.value, "tiles": t.value}


def aio_linear_pack(h: int, W_rowmajor: int, scales, W_packed: int, scales_packed, stream: int = 0):
    _check(_lib.aio_linear_pack(h, W_rowmajor, scales, W_packed, scales_packed, stream), "aio_linear_pack")


def aio_linear_unpack(h: int, W_packed: int, W_rowmajor: int, stream: int = 0):
    _check(_lib.aio_linear_unpack(h, W_packed, W_rowmajor, stream), "aio_linear_unpack")


def aio_linear_run(h: int, x: int, M: int, K: int, N: int, W: int, scales, y: int, stream: int = 0):
    _check(_lib.aio_linear_run(h, x, M, K, N, W, scales, y, stream), "aio_linear_run")


def aio_linear_run_noalloc(x: int, M: int, K: int, N: int, wt: int, flags: int, W: int, scales, y: int,
                           device_error: int, stream: int = 0):
    _check(_lib.aio_linear_run_noalloc(x, M, K, N, wt, flags, W, scales, y, device_error, stream),
           "aio_linear_run_noalloc")


def aio_linear_check(h: int) -> int:
    e = _int()
    _check(_lib.aio_linear_check(h, ctypes.byref(e)), "aio_linear_check")
    return e.value


def aio_linear_reset(h: int):
    _check(_lib.aio_linear_reset(h), "aio_linear_reset")


def aio_linear_destroy(h: int):
    _check(_lib.aio_linear_destroy(h), "aio_linear_destroy")


def aio_decode_step_create(projs, M: int, flags: int = AIO_STEP_GRAPH | AIO_STEP_PERSISTENT) -> int:
    """projs: sequence of (h, x, W, scales, y) integer addresses (scales may be None)."""
    arr = (aio_proj * len(projs))(*[aio_proj(*p) for p in projs])
    s = _vp()
    _check(_lib.aio_decode_step_create(ctypes.byref(s), arr, len(projs), M, flags), "aio_decode_step_create")
    return s.value


def aio_decode_step_create_chained(projs, preps, M: int, flags: int = AIO_STEP_GRAPH | AIO_STEP_PERSISTENT) -> int:
    """projs as for aio_decode_step_create; preps: one (op, src, src_stride, src_off, h_in, h_out,
    gamma, eps[, kv_cache, L_past, n_heads, L_max]) tuple per projection, addresses as integers or
    None."""
    assert len(preps) == len(projs)
    arr = (aio_proj * len(projs))(*[aio_proj(*p) for p in projs])
    parr = (aio_xprep * len(preps))(*[aio_xprep(*x) for x in preps])
    s = _vp()
    _check(_lib.aio_decode_step_create_chained(ctypes.byref(s), arr, parr, len(projs), M, flags),
           "aio_decode_step_create_chained")
    return s.value


def aio_decode_step(step: int, stream: int = 0):
    _check(_lib.aio_decode_step(step, stream), "aio_decode_step")


def aio_decode_step_host(step: int, x_host: int, x_dev: int, x_bytes: int, y_dev: int, y_host: int, y_bytes: int,
                         stream: int = 0):
    _check(_lib.aio_decode_step_host(step, x_host, x_dev, x_bytes, y_dev, y_host, y_bytes, stream),
           "aio_decode_step_host")


def aio_decode_step_kernels(step: int) -> int:
    n = _int()
    _check(_lib.aio_decode_step_kernels(step, ctypes.byref(n)), "aio_decode_step_kernels")
    return n.value


def aio_decode_step_check(step: int) -> int:
    e = _int()
    _check(_lib.aio_decode_step_check(step, ctypes.byref(e)), "aio_decode_step_check")
    return e.value


def aio_decode_step_reset(step: int):
    _check(_lib.aio_decode_step_reset(step), "aio_decode_step_reset")


def aio_decode_step_destroy(step: int):
    _check(_lib.aio_decode_step_destroy(step), "aio_decode_step_destroy")


def aio_probe_read(buf: int, nbytes: int, out: int, stream: int = 0):
    _check(_lib.aio_probe_read(buf, nbytes, out, stream), "aio_probe_read")


def aio_attention_workspace_bytes(M: int) -> int:
    b = _sz()
    _check(_lib.aio_attention_workspace_bytes(M, ctypes.byref(b)), "aio_attention_workspace_bytes")
    return b.value


def aio_attention_decode(q: int, q_stride: int, k_cache: int, v_cache: int, n_heads: int, head_dim: int, L_max: int,
                         L: int, M: int, out: int, workspace: int, workspace_bytes: int, stream: int = 0):
    _check(_lib.aio_attention_decode(q, q_stride, k_cache, v_cache, n_heads, head_dim, L_max, L, M, out, workspace,
                                     workspace_bytes, stream), "aio_attention_decode")


def aio_attention_check(workspace: int) -> int:
    e = _int()
    _check(_lib.aio_attention_check(workspace, ctypes.byref(e)), "aio_attention_check")
    return e.value


def aio_pld_draft(tokens: int, T: int, N: int, L: int, out: int, stream: int = 0):
    _check(_lib.aio_pld_draft(tokens, T, N, L, out, stream), "aio_pld_draft")


def aio_argmax_rows(logits: int, M: int, V: int, stride: int, out: int, stream: int = 0):
    _check(_lib.aio_argmax_rows(logits, M, V, stride, out, stream), "aio_argmax_rows")


def aio_pld_accept(argmax: int, draft: int, result: int, stream: int = 0):
    _check(_lib.aio_pld_accept(argmax, draft, result, stream), "aio_pld_accept")


def aio_route(logits: int, category_tokens: int, n_categories: int, code_index: int, L_ctx: int, tau: float,
              decision: int, stream: int = 0):
    _check(_lib.aio_route(logits, category_tokens, n_categories, code_index, L_ctx, tau, decision, stream), "aio_route")
