"""ctypes binding of librowop (``include/rowop.h``).

Two layers, both argument marshalling only -- every step of the computation
runs in the CUDA library:

* ``rowop_*`` functions with the C names and C arguments (integers for
  pointers and streams), returning the C status code;
* tensor helpers (``softmax``, ``layernorm_ragged``, ...) that take CUDA torch
  tensors, allocate outputs / workspace with torch, pass
  ``data_ptr()`` and the current stream, and raise ``RowopError`` on a
  non-OK status.

There is no fallback: if the shared library has not been built the first
call raises, and a tensor that is not on a CUDA device is rejected.
"""
from __future__ import annotations

import ctypes
import os
import threading

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "_build", "librowop.so")

ROWOP_F32, ROWOP_BF16, ROWOP_F16 = 0, 1, 2
SMALL, MEDIUM, LARGE = 0, 1, 2
STATUS = {
    0: "ROWOP_OK", 1: "ROWOP_ERR_INVALID_ARG", 2: "ROWOP_ERR_UNSUPPORTED_DTYPE",
    3: "ROWOP_ERR_WORKSPACE", 4: "ROWOP_ERR_CUDA", 5: "ROWOP_ERR_TIMEOUT",
    6: "ROWOP_ERR_BAD_OFFSETS", 7: "ROWOP_ERR_TOO_LONG",
}
globals().update({v: k for k, v in STATUS.items()})

_lock = threading.Lock()
_lib = None

_P = ctypes.c_void_p
_I64 = ctypes.c_int64
_I = ctypes.c_int
_F = ctypes.c_float
_SZ = ctypes.c_size_t

class RowopConfig(ctypes.Structure):
    """rowop_config_t of include/rowop.h."""
    _fields_ = [("size", ctypes.c_uint32), ("chunk_bytes", ctypes.c_uint32),
                ("tile_bytes", ctypes.c_uint32), ("max_cluster", ctypes.c_uint32),
                ("small_max_bytes", _I64), ("medium_max_bytes", _I64),
                ("max_row_len", _I64 * 3), ("resident_max_tiles", _I64 * 2),
                ("staged_max_tiles", _I64), ("stage_budget_bytes", _I64 * 2),
                ("wait_limit_ns", _I64), ("static_max_rows", _I64)]


# C signatures (argument types, return type), in header order.
SIGNATURES = {
    "rowop_softmax": ([_P, _P, _I64, _I64, _I64, _I, _P], _I),
    "rowop_logsoftmax": ([_P, _P, _I64, _I64, _I64, _I, _P], _I),
    "rowop_layernorm": ([_P, _P, _P, _P, _I64, _I64, _I64, _I, _F, _P], _I),
    "rowop_rmsnorm": ([_P, _P, _P, _I64, _I64, _I64, _I, _F, _P], _I),
    "rowop_ragged_workspace_size": ([_I64], _SZ),
    "rowop_softmax_ragged": ([_P, _P, _P, _I64, _I64, _I, _P, _SZ, _P], _I),
    "rowop_logsoftmax_ragged": ([_P, _P, _P, _I64, _I64, _I, _P, _SZ, _P], _I),
    "rowop_layernorm_ragged": ([_P, _P, _P, _P, _P, _I64, _I64, _I, _F, _P, _SZ, _P], _I),
    "rowop_rmsnorm_ragged": ([_P, _P, _P, _P, _I64, _I64, _I, _F, _P, _SZ, _P], _I),
    "rowop_ragged_plan": ([_P, _I64, _I64, _I, _P, _SZ, _P], _I),
    "rowop_softmax_ragged_planned": ([_P, _P, _P, _I64, _I64, _I, _P, _SZ, _P], _I),
    "rowop_logsoftmax_ragged_planned": ([_P, _P, _P, _I64, _I64, _I, _P, _SZ, _P], _I),
    "rowop_layernorm_ragged_planned": ([_P, _P, _P, _P, _P, _I64, _I64, _I, _F, _P, _SZ,
                                        _P], _I),
    "rowop_rmsnorm_ragged_planned": ([_P, _P, _P, _P, _I64, _I64, _I, _F, _P, _SZ, _P], _I),
    "rowop_layernorm_ragged_static": ([_P, _P, _P, _P, _P, _I64, _I64, _I, _F, _P], _I),
    "rowop_add_layernorm": ([_P, _P, _P, _P, _P, _P, _I64, _I64, _I64, _I, _F, _P], _I),
    "rowop_add_rmsnorm": ([_P, _P, _P, _P, _P, _I64, _I64, _I64, _I, _F, _P], _I),
    "rowop_softmax_backward": ([_P, _P, _P, _I64, _I64, _I64, _I, _P], _I),
    "rowop_logsoftmax_backward": ([_P, _P, _P, _I64, _I64, _I64, _I, _P], _I),
    "rowop_layernorm_backward": ([_P, _P, _P, _P, _P, _P, _I64, _I64, _I64, _I, _F, _P, _SZ,
                                  _P], _I),
    "rowop_rmsnorm_backward": ([_P, _P, _P, _P, _P, _I64, _I64, _I64, _I, _F, _P, _SZ, _P], _I),
    "rowop_softmax_backward_ragged": ([_P, _P, _P, _P, _I64, _I64, _I, _P, _SZ, _P], _I),
    "rowop_logsoftmax_backward_ragged": ([_P, _P, _P, _P, _I64, _I64, _I, _P, _SZ, _P], _I),
    "rowop_layernorm_backward_ragged": ([_P, _P, _P, _P, _P, _P, _P, _I64, _I64, _I, _F, _P,
                                         _SZ, _P], _I),
    "rowop_rmsnorm_backward_ragged": ([_P, _P, _P, _P, _P, _P, _I64, _I64, _I, _F, _P, _SZ, _P],
                                      _I),
    "rowop_layernorm_backward_ragged_workspace_size": ([_I64, _I64, _I], _SZ),
    "rowop_rmsnorm_backward_ragged_workspace_size": ([_I64, _I64, _I], _SZ),
    "rowop_layernorm_backward_workspace_size": ([_I64], _SZ),
    "rowop_rmsnorm_backward_workspace_size": ([_I64], _SZ),
    "rowop_pad_scale": ([_P, _P, _I64, _I64, _I64, _I64, _I64, _F, _I, _P], _I),
    "rowop_moe_group_top2": ([_P, _P, _I64, _I64, _I64, _I, _P], _I),
    "rowop_select_bucket": ([_I64, _I], _I),
    "rowop_max_row_len": ([_I], _I64),
    "rowop_get_config": ([ctypes.POINTER(RowopConfig)], _I),
    "rowop_status_string": ([_I], ctypes.c_char_p),
    "rowop_last_cuda_error": ([], ctypes.c_char_p),
    "rowop_check_status": ([_P], _I),
    "rowop_debug_wait_timeout": ([_I64, _P], _I),
}


class RowopError(RuntimeError):
    def __init__(self, status: int, what: str = ""):
        self.status = status
        super().__init__(f"{what}: {STATUS.get(status, status)}" if what else
                         STATUS.get(status, str(status)))


def load(path: str | None = None) -> ctypes.CDLL:
    """Loads librowop.so (built by ``build.build()``); raises if it is missing."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        p = path or LIB_PATH
        if not os.path.exists(p):
            raise RuntimeError(
                f"librowop is not built ({p} missing): run "
                "paper_2607_23089_gb300.build.build() first")
        lib = ctypes.CDLL(p)
        for name, (argtypes, restype) in SIGNATURES.items():
            fn = getattr(lib, name)
            fn.argtypes = argtypes
            fn.restype = restype
        _lib = lib
        return lib


def _c(name):
    def call(*args):
        return getattr(load(), name)(*args)
    call.__name__ = name
    call.__doc__ = f"Direct call of the C function {name} (see include/rowop.h)."
    return call


for _name in SIGNATURES:
    globals()[_name] = _c(_name)


def get_config() -> dict:
    """rowop_get_config() as a dict."""
    cfg = RowopConfig()
    st = rowop_get_config(ctypes.byref(cfg))  # noqa: F821 (defined above)
    if st != 0:
        raise RowopError(st, "rowop_get_config")
    out = {}
    for name, _ in RowopConfig._fields_:
        v = getattr(cfg, name)
        out[name] = list(v) if hasattr(v, "__len__") else int(v)
    return out


# ---------------------------------------------------------------------------
# torch tensor helpers
# ---------------------------------------------------------------------------
def _torch():
    import torch
    return torch


def dtype_code(dtype) -> int:
    torch = _torch()
    if dtype == torch.float32:
        return ROWOP_F32
    if dtype == torch.bfloat16:
        return ROWOP_BF16
    if dtype == torch.float16:
        return ROWOP_F16
    raise TypeError(f"librowop supports float32, bfloat16 and float16, not {dtype}")


def _stream(stream):
    if stream is None:
        return _torch().cuda.current_stream().cuda_stream
    return getattr(stream, "cuda_stream", stream)


def _ptr(t):
    return None if t is None else t.data_ptr()


def _check_cuda(*ts):
    for t in ts:
        if t is not None and not t.is_cuda:
            raise ValueError("librowop operates on CUDA tensors only")


def _ok(st, what):
    if st != 0:
        if st == ROWOP_ERR_CUDA:
            what = f"{what} ({_lib.rowop_last_cuda_error().decode()})"
        raise RowopError(st, what)


def _dense_layout(x):
    if x.dim() != 2:
        raise ValueError("dense ops take a 2-D rows x cols tensor")
    rows, cols = x.shape
    if cols > 1 and x.stride(1) != 1:
        raise ValueError("rows must be contiguous (stride(1) == 1)")
    ld = x.stride(0) if rows > 1 else cols
    return rows, cols, max(ld, cols)


def _out_like(x, out):
    if out is None:
        out = _torch().empty_strided(x.shape, x.stride(), dtype=x.dtype, device=x.device)
    elif out.shape != x.shape or out.stride() != x.stride() or out.dtype != x.dtype:
        raise ValueError("out must match x in shape, strides and dtype")
    return out


def softmax(x, out=None, stream=None):
    _check_cuda(x, out)
    rows, cols, ld = _dense_layout(x)
    out = _out_like(x, out)
    _ok(rowop_softmax(x.data_ptr(), out.data_ptr(), rows, cols, ld,  # noqa: F821
                      dtype_code(x.dtype), _stream(stream)), "rowop_softmax")
    return out


def logsoftmax(x, out=None, stream=None):
    _check_cuda(x, out)
    rows, cols, ld = _dense_layout(x)
    out = _out_like(x, out)
    _ok(rowop_logsoftmax(x.data_ptr(), out.data_ptr(), rows, cols, ld,  # noqa: F821
                         dtype_code(x.dtype), _stream(stream)), "rowop_logsoftmax")
    return out


def layernorm(x, gamma=None, beta=None, eps=1e-5, out=None, stream=None):
    _check_cuda(x, gamma, beta, out)
    rows, cols, ld = _dense_layout(x)
    out = _out_like(x, out)
    _ok(rowop_layernorm(x.data_ptr(), out.data_ptr(), _ptr(gamma), _ptr(beta),  # noqa: F821
                        rows, cols, ld, dtype_code(x.dtype), float(eps),
                        _stream(stream)), "rowop_layernorm")
    return out


def rmsnorm(x, gamma=None, eps=1e-6, out=None, stream=None):
    _check_cuda(x, gamma, out)
    rows, cols, ld = _dense_layout(x)
    out = _out_like(x, out)
    _ok(rowop_rmsnorm(x.data_ptr(), out.data_ptr(), _ptr(gamma), rows, cols,  # noqa: F821
                      ld, dtype_code(x.dtype), float(eps), _stream(stream)),
        "rowop_rmsnorm")
    return out


def ragged_workspace(rows: int, device="cuda"):
    """A workspace tensor for a ragged call over ``rows`` rows."""
    n = rowop_ragged_workspace_size(int(rows))  # noqa: F821
    return _torch().empty(int(n), dtype=_torch().uint8, device=device)


def _ragged_args(x, offsets, ws, out):
    _check_cuda(x, offsets, ws, out)
    torch = _torch()
    if offsets.dtype != torch.int64 or offsets.dim() != 1:
        raise ValueError("offsets must be a 1-D int64 tensor")
    rows = offsets.numel() - 1
    if out is None:
        out = torch.empty_like(x)
    if ws is None:
        ws = ragged_workspace(rows, x.device)
    return rows, out, ws


def softmax_ragged(x, offsets, max_len, out=None, ws=None, stream=None):
    rows, out, ws = _ragged_args(x, offsets, ws, out)
    _ok(rowop_softmax_ragged(x.data_ptr(), out.data_ptr(), offsets.data_ptr(),  # noqa: F821
                             rows, int(max_len), dtype_code(x.dtype), ws.data_ptr(),
                             ws.numel(), _stream(stream)), "rowop_softmax_ragged")
    return out


def logsoftmax_ragged(x, offsets, max_len, out=None, ws=None, stream=None):
    rows, out, ws = _ragged_args(x, offsets, ws, out)
    _ok(rowop_logsoftmax_ragged(x.data_ptr(), out.data_ptr(),  # noqa: F821
                                offsets.data_ptr(), rows, int(max_len),
                                dtype_code(x.dtype), ws.data_ptr(), ws.numel(),
                                _stream(stream)), "rowop_logsoftmax_ragged")
    return out


def layernorm_ragged(x, offsets, max_len, gamma=None, beta=None, eps=1e-5,
                     out=None, ws=None, stream=None):
    _check_cuda(gamma, beta)
    rows, out, ws = _ragged_args(x, offsets, ws, out)
    _ok(rowop_layernorm_ragged(x.data_ptr(), out.data_ptr(), _ptr(gamma),  # noqa: F821
                               _ptr(beta), offsets.data_ptr(), rows, int(max_len),
                               dtype_code(x.dtype), float(eps), ws.data_ptr(),
                               ws.numel(), _stream(stream)), "rowop_layernorm_ragged")
    return out


def rmsnorm_ragged(x, offsets, max_len, gamma=None, eps=1e-6, out=None, ws=None,
                   stream=None):
    _check_cuda(gamma)
    rows, out, ws = _ragged_args(x, offsets, ws, out)
    _ok(rowop_rmsnorm_ragged(x.data_ptr(), out.data_ptr(), _ptr(gamma),  # noqa: F821
                             offsets.data_ptr(), rows, int(max_len),
                             dtype_code(x.dtype), float(eps), ws.data_ptr(),
                             ws.numel(), _stream(stream)), "rowop_rmsnorm_ragged")
    return out


def check_status(stream=None) -> int:
    """Synchronises the stream and returns (and clears) the device status."""
    return rowop_check_status(_stream(stream))  # noqa: F821


def select_bucket(length: int, dtype) -> int:
    code = dtype if isinstance(dtype, int) else dtype_code(dtype)
    return rowop_select_bucket(int(length), code)  # noqa: F821


def add_layernorm(x, r, gamma=None, beta=None, eps=1e-5, sum_out=None, out=None, stream=None):
    """Fused residual add + LayerNorm (``rowop_add_layernorm``): returns
    ``(x + r, LayerNorm(x + r))``."""
    torch = _torch()
    _check_cuda(x, r, gamma, beta)
    rows, cols = x.shape
    sum_out = torch.empty_like(x) if sum_out is None else sum_out
    out = torch.empty_like(x) if out is None else out
    _ok(rowop_add_layernorm(x.data_ptr(), r.data_ptr(), sum_out.data_ptr(),  # noqa: F821
                            out.data_ptr(), _ptr(gamma), _ptr(beta), rows, cols, x.stride(0),
                            dtype_code(x.dtype), float(eps), _stream(stream)),
        "rowop_add_layernorm")
    return sum_out, out


def add_rmsnorm(x, r, gamma=None, eps=1e-6, sum_out=None, out=None, stream=None):
    """Fused residual add + RMSNorm (``rowop_add_rmsnorm``): returns
    ``(x + r, RMSNorm(x + r))``."""
    torch = _torch()
    _check_cuda(x, r, gamma)
    rows, cols = x.shape
    sum_out = torch.empty_like(x) if sum_out is None else sum_out
    out = torch.empty_like(x) if out is None else out
    _ok(rowop_add_rmsnorm(x.data_ptr(), r.data_ptr(), sum_out.data_ptr(),  # noqa: F821
                          out.data_ptr(), _ptr(gamma), rows, cols, x.stride(0),
                          dtype_code(x.dtype), float(eps), _stream(stream)),
        "rowop_add_rmsnorm")
    return sum_out, out


def pad_scale(x, fft_size: int, scale: float, out=None, stream=None):
    """Hyena FFT-size padding of a rows x seqlen tensor to rows x fft_size
    (``rowop_pad_scale``)."""
    torch = _torch()
    _check_cuda(x)
    rows, seqlen = x.shape
    if out is None:
        out = torch.empty((rows, fft_size), dtype=x.dtype, device=x.device)
    _ok(rowop_pad_scale(x.data_ptr(), out.data_ptr(), rows, seqlen, int(fft_size),  # noqa: F821
                        x.stride(0), out.stride(0), float(scale), dtype_code(x.dtype),
                        _stream(stream)), "rowop_pad_scale")
    return out


def moe_group_top2(scores, out=None, stream=None):
    """Per-group sum of the two largest of every 32 consecutive expert scores,
    float32 (``rowop_moe_group_top2``)."""
    torch = _torch()
    _check_cuda(scores)
    tokens, experts = scores.shape
    if out is None:
        out = torch.empty((tokens, experts // 32), dtype=torch.float32, device=scores.device)
    _ok(rowop_moe_group_top2(scores.data_ptr(), out.data_ptr(), tokens, experts,  # noqa: F821
                             scores.stride(0), dtype_code(scores.dtype), _stream(stream)),
        "rowop_moe_group_top2")
    return out


def softmax_backward(y, dy, dx=None, stream=None):
    """dx of softmax from its output y and the upstream gradient dy
    (``rowop_softmax_backward``)."""
    _check_cuda(y, dy, dx)
    rows, cols, ld = _dense_layout(y)
    dx = _out_like(y, dx)
    _ok(rowop_softmax_backward(y.data_ptr(), dy.data_ptr(), dx.data_ptr(), rows, cols,  # noqa: F821
                               ld, dtype_code(y.dtype), _stream(stream)),
        "rowop_softmax_backward")
    return dx


def logsoftmax_backward(y, dy, dx=None, stream=None):
    """dx of log-softmax from its output y and dy (``rowop_logsoftmax_backward``)."""
    _check_cuda(y, dy, dx)
    rows, cols, ld = _dense_layout(y)
    dx = _out_like(y, dx)
    _ok(rowop_logsoftmax_backward(y.data_ptr(), dy.data_ptr(), dx.data_ptr(), rows,  # noqa: F821
                                  cols, ld, dtype_code(y.dtype), _stream(stream)),
        "rowop_logsoftmax_backward")
    return dx


def softmax_backward_ragged(y, dy, offsets, max_len, dx=None, ws=None, stream=None,
                            log=False):
    """dx of softmax (log-softmax with ``log=True``) over ragged rows
    (``rowop_{softmax,logsoftmax}_backward_ragged``)."""
    rows, dx, ws = _ragged_args(y, offsets, ws, dx)
    _check_cuda(dy)
    fn = rowop_logsoftmax_backward_ragged if log else rowop_softmax_backward_ragged  # noqa: F821
    _ok(fn(y.data_ptr(), dy.data_ptr(), dx.data_ptr(), offsets.data_ptr(), rows, int(max_len),
           dtype_code(y.dtype), ws.data_ptr(), ws.numel(), _stream(stream)),
        "rowop_softmax_backward_ragged")
    return dx


def _bwd_params(x, want, given, ws, size_fn):
    torch = _torch()
    cols = x.shape[1]
    outs = [g if g is not None else (torch.empty(cols, dtype=x.dtype, device=x.device)
                                     if w else None) for w, g in zip(want, given)]
    if any(o is not None for o in outs) and ws is None:
        ws = torch.empty(int(size_fn(cols)), dtype=torch.uint8, device=x.device)
    return outs, ws


def layernorm_backward(x, dy, gamma=None, eps=1e-5, want_dgamma=True, want_dbeta=True,
                       dx=None, dgamma=None, dbeta=None, ws=None, stream=None):
    """LayerNorm backward from the forward input x (``rowop_layernorm_backward``):
    returns ``(dx, dgamma, dbeta)``, the last two None when not wanted (given
    output tensors are used as they are)."""
    _check_cuda(x, dy, gamma, dx, dgamma, dbeta, ws)
    rows, cols, ld = _dense_layout(x)
    dx = _out_like(x, dx)
    (dg, db), ws = _bwd_params(x, (want_dgamma, want_dbeta), (dgamma, dbeta), ws,
                               rowop_layernorm_backward_workspace_size)  # noqa: F821
    _ok(rowop_layernorm_backward(x.data_ptr(), dy.data_ptr(), _ptr(gamma), dx.data_ptr(),  # noqa: F821
                                 _ptr(dg), _ptr(db), rows, cols, ld, dtype_code(x.dtype),
                                 float(eps), _ptr(ws), 0 if ws is None else ws.numel(),
                                 _stream(stream)), "rowop_layernorm_backward")
    return dx, dg, db


def rmsnorm_backward(x, dy, gamma=None, eps=1e-6, want_dgamma=True, dx=None, dgamma=None,
                     ws=None, stream=None):
    """RMSNorm backward from the forward input x (``rowop_rmsnorm_backward``):
    returns ``(dx, dgamma)``, dgamma None when not wanted."""
    _check_cuda(x, dy, gamma, dx, dgamma, ws)
    rows, cols, ld = _dense_layout(x)
    dx = _out_like(x, dx)
    (dg,), ws = _bwd_params(x, (want_dgamma,), (dgamma,), ws,
                            rowop_rmsnorm_backward_workspace_size)  # noqa: F821
    _ok(rowop_rmsnorm_backward(x.data_ptr(), dy.data_ptr(), _ptr(gamma), dx.data_ptr(),  # noqa: F821
                               _ptr(dg), rows, cols, ld, dtype_code(x.dtype), float(eps),
                               _ptr(ws), 0 if ws is None else ws.numel(), _stream(stream)),
        "rowop_rmsnorm_backward")
    return dx, dg


def _ragged_norm_backward(x, dy, offsets, max_len, gamma, eps, want, given, dx, ws, stream,
                          size_fn, call, name):
    torch = _torch()
    _check_cuda(x, dy, offsets, gamma, dx, ws, *given)
    rows = offsets.numel() - 1
    max_len = int(max_len)
    dx = torch.empty_like(x) if dx is None else dx
    outs = [g if g is not None else (torch.empty(max_len, dtype=x.dtype, device=x.device)
                                     if w else None) for w, g in zip(want, given)]
    code = dtype_code(x.dtype)
    if ws is None:
        ws = torch.empty(int(size_fn(rows, max_len, code)), dtype=torch.uint8, device=x.device)
    _ok(call(x.data_ptr(), dy.data_ptr(), _ptr(gamma), dx.data_ptr(), *[_ptr(o) for o in outs],
             offsets.data_ptr(), rows, max_len, code, float(eps), ws.data_ptr(), ws.numel(),
             _stream(stream)), name)
    return (dx, *outs)


def layernorm_backward_ragged(x, dy, offsets, max_len, gamma=None, eps=1e-5, want_dgamma=True,
                              want_dbeta=True, dx=None, dgamma=None, dbeta=None, ws=None,
                              stream=None):
    """LayerNorm backward over ragged rows (``rowop_layernorm_backward_ragged``):
    returns ``(dx, dgamma, dbeta)``, dgamma / dbeta of max_len elements or
    None when not wanted."""
    return _ragged_norm_backward(
        x, dy, offsets, max_len, gamma, eps, (want_dgamma, want_dbeta), (dgamma, dbeta), dx, ws,
        stream, rowop_layernorm_backward_ragged_workspace_size,  # noqa: F821
        rowop_layernorm_backward_ragged, "rowop_layernorm_backward_ragged")  # noqa: F821


def rmsnorm_backward_ragged(x, dy, offsets, max_len, gamma=None, eps=1e-6, want_dgamma=True,
                            dx=None, dgamma=None, ws=None, stream=None):
    """RMSNorm backward over ragged rows (``rowop_rmsnorm_backward_ragged``):
    returns ``(dx, dgamma)``."""
    return _ragged_norm_backward(
        x, dy, offsets, max_len, gamma, eps, (want_dgamma,), (dgamma,), dx, ws, stream,
        rowop_rmsnorm_backward_ragged_workspace_size,  # noqa: F821
        rowop_rmsnorm_backward_ragged, "rowop_rmsnorm_backward_ragged")  # noqa: F821


def run(op: str, x, *, offsets=None, max_len=None, gamma=None, beta=None,
        eps=None, out=None, ws=None, stream=None, fft_size=None, scale=None, resid=None,
        sum_out=None, dy=None, dgamma=None, dbeta=None):
    """One call of ``op`` on dense or ragged input (ragged when offsets is
    given); returns the output tensor (dx for the backward passes, whose x is
    the forward output for the softmax family and the forward input for the
    norms)."""
    if offsets is not None and op in ("pad_scale", "add_layernorm", "add_rmsnorm",
                                      "moe_group_top2"):
        raise ValueError(f"{op} has no ragged form")
    if offsets is not None and op.endswith("_backward"):
        if op in ("softmax_backward", "logsoftmax_backward"):
            return softmax_backward_ragged(x, dy, offsets, max_len, dx=out, ws=ws, stream=stream,
                                           log=op.startswith("log"))
        if op == "layernorm_backward":
            return layernorm_backward_ragged(x, dy, offsets, max_len, gamma,
                                             1e-5 if eps is None else eps, dx=out, dgamma=dgamma,
                                             dbeta=dbeta, ws=ws, stream=stream)[0]
        if op == "rmsnorm_backward":
            return rmsnorm_backward_ragged(x, dy, offsets, max_len, gamma,
                                           1e-6 if eps is None else eps, dx=out, dgamma=dgamma,
                                           ws=ws, stream=stream)[0]
    if op == "softmax_backward":
        return softmax_backward(x, dy, out, stream)
    if op == "logsoftmax_backward":
        return logsoftmax_backward(x, dy, out, stream)
    if op == "layernorm_backward":
        return layernorm_backward(x, dy, gamma, 1e-5 if eps is None else eps,
                                  want_dgamma=True, want_dbeta=True, dx=out, dgamma=dgamma,
                                  dbeta=dbeta, ws=ws, stream=stream)[0]
    if op == "rmsnorm_backward":
        return rmsnorm_backward(x, dy, gamma, 1e-6 if eps is None else eps, want_dgamma=True,
                                dx=out, dgamma=dgamma, ws=ws, stream=stream)[0]
    if op == "pad_scale":
        return pad_scale(x, fft_size, scale, out, stream)
    if op == "add_layernorm":
        return add_layernorm(x, resid, gamma, beta, 1e-5 if eps is None else eps, sum_out, out,
                             stream)[1]
    if op == "add_rmsnorm":
        return add_rmsnorm(x, resid, gamma, 1e-6 if eps is None else eps, sum_out, out, stream)[1]
    if op == "moe_group_top2":
        return moe_group_top2(x, out, stream)
    if offsets is None:
        if op == "softmax":
            return softmax(x, out, stream)
        if op == "logsoftmax":
            return logsoftmax(x, out, stream)
        if op == "layernorm":
            return layernorm(x, gamma, beta, 1e-5 if eps is None else eps, out, stream)
        if op == "rmsnorm":
            return rmsnorm(x, gamma, 1e-6 if eps is None else eps, out, stream)
    else:
        if op == "softmax":
            return softmax_ragged(x, offsets, max_len, out, ws, stream)
        if op == "logsoftmax":
            return logsoftmax_ragged(x, offsets, max_len, out, ws, stream)
        if op == "layernorm":
            return layernorm_ragged(x, offsets, max_len, gamma, beta,
                                    1e-5 if eps is None else eps, out, ws, stream)
        if op == "rmsnorm":
            return rmsnorm_ragged(x, offsets, max_len, gamma,
                                  1e-6 if eps is None else eps, out, ws, stream)
    raise ValueError(f"unknown op {op}")
