"""Python face of the double-precision CPU oracle (``rowop_oracle.c``).

TEST INFRASTRUCTURE ONLY.  This module is the oracle the CUDA library is
compared against.  Only the test suite, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline / reference leg may import it; the product path
(``paper_2607_23089_gb300``) never does, and this module never imports the
product.  Inputs arrive here as exact float64 copies of whatever the GPU saw
(bf16 and fp32 values convert to double without rounding), outputs leave as
float64.

Definitions (textbook / PyTorch convention; the paper names the family only
through its running-example kernel names in §2.1 and writes no formula):

* softmax     ``y = exp(x - max x) / sum exp(x - max x)``
* log-softmax ``y = (x - max x) - log(sum exp(x - max x))``
* LayerNorm   ``y = (x - mu) / sqrt(var + eps) * gamma + beta`` with the biased
  (population) variance
* RMSNorm     ``y = x / sqrt(mean(x^2) + eps) * gamma``
* ragged      row ``i`` is ``x[off[i]:off[i+1]]``; gamma/beta are indexed by the
  column inside the row.

``eps`` is passed as the float32 value the GPU uses, widened to double.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "rowop_oracle.c")
_SRCS = [_SRC, os.path.join(_HERE, "pad_moe_oracle.c"), os.path.join(_HERE, "backward_oracle.c")]
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "liboracle.so")
_lock = threading.Lock()
_lib = None

SMALL, MEDIUM, LARGE = 0, 1, 2


def build(force: bool = False) -> str:
    """Compile ``rowop_oracle.c``, ``pad_moe_oracle.c`` and
    ``backward_oracle.c`` with gcc (-O2, no fast-math) into a shared library next to them.  OpenMP is used when the
    compiler offers it; without it the row loop simply runs on one thread."""
    os.makedirs(_BUILD_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and all(os.path.getmtime(_LIB_PATH) >= os.path.getmtime(s) for s in _SRCS)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    base = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fno-fast-math",
            "-ffp-contract=off", *_SRCS, "-o", tmp, "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True,
                       capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = ctypes.CDLL(build())
        d, i64, ci = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int
        dbl = ctypes.c_double
        lib.oracle_softmax.argtypes = [d, d, i64, i64, ci]
        lib.oracle_logsoftmax.argtypes = [d, d, i64, i64, ci]
        lib.oracle_layernorm.argtypes = [d, d, d, d, i64, i64, dbl, ci]
        lib.oracle_rmsnorm.argtypes = [d, d, d, i64, i64, dbl, ci]
        lib.oracle_softmax_ragged.argtypes = [d, d, d, i64, ci]
        lib.oracle_logsoftmax_ragged.argtypes = [d, d, d, i64, ci]
        lib.oracle_layernorm_ragged.argtypes = [d, d, d, d, d, i64, dbl, ci]
        lib.oracle_rmsnorm_ragged.argtypes = [d, d, d, d, i64, dbl, ci]
        lib.oracle_bucket.argtypes = [i64, i64]
        lib.oracle_bucket.restype = ci
        lib.oracle_pad_scale.argtypes = [d, d, i64, i64, i64, dbl]
        lib.oracle_moe_group_top2.argtypes = [d, d, i64, i64, i64]
        lib.oracle_softmax_backward.argtypes = [d, d, d, i64, i64, ci]
        lib.oracle_logsoftmax_backward.argtypes = [d, d, d, i64, i64, ci]
        lib.oracle_layernorm_backward.argtypes = [d, d, d, d, d, d, i64, i64, dbl, ci]
        lib.oracle_layernorm_backward.restype = ci
        lib.oracle_rmsnorm_backward.argtypes = [d, d, d, d, d, i64, i64, dbl, ci]
        lib.oracle_rmsnorm_backward.restype = ci
        lib.oracle_softmax_backward.restype = None
        lib.oracle_logsoftmax_backward.restype = None
        for name in ("oracle_softmax", "oracle_logsoftmax", "oracle_layernorm",
                     "oracle_rmsnorm", "oracle_softmax_ragged",
                     "oracle_logsoftmax_ragged", "oracle_layernorm_ragged",
                     "oracle_rmsnorm_ragged", "oracle_pad_scale",
                     "oracle_moe_group_top2"):
            getattr(lib, name).restype = None
        _lib = lib
        return lib


def _f64(a) -> np.ndarray:
    a = np.asarray(a, dtype=np.float64)
    return np.ascontiguousarray(a)


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _threads(nthreads):
    return int(nthreads) if nthreads else 1


def _as_eps(eps: float) -> float:
    # The GPU adds eps as a float32; the oracle uses that same value.
    return float(np.float32(eps))


def _dense(name, x, nthreads, *extra_arrays, eps=None):
    x = _f64(x)
    if x.ndim != 2:
        raise ValueError("dense oracle wants a 2-D rows x cols array")
    rows, cols = x.shape
    y = np.empty_like(x)
    lib = _load()
    args = [_ptr(x), _ptr(y)] + [_ptr(a) for a in extra_arrays]
    args += [rows, cols]
    if eps is not None:
        args.append(_as_eps(eps))
    args.append(_threads(nthreads))
    getattr(lib, name)(*args)
    return y


def _vec(v, n, fill):
    if v is None:
        return np.full(n, fill, dtype=np.float64)
    v = _f64(v).reshape(-1)
    if v.shape[0] < n:
        raise ValueError("gamma/beta shorter than the row length")
    return v


def softmax(x, nthreads=1):
    return _dense("oracle_softmax", x, nthreads)


def logsoftmax(x, nthreads=1):
    return _dense("oracle_logsoftmax", x, nthreads)


def layernorm(x, gamma=None, beta=None, eps=1e-5, nthreads=1):
    x = _f64(x)
    n = x.shape[1]
    return _dense("oracle_layernorm", x, nthreads, _vec(gamma, n, 1.0),
                  _vec(beta, n, 0.0), eps=eps)


def rmsnorm(x, gamma=None, eps=1e-6, nthreads=1):
    x = _f64(x)
    n = x.shape[1]
    return _dense("oracle_rmsnorm", x, nthreads, _vec(gamma, n, 1.0), eps=eps)


def _offsets(offsets):
    off = np.ascontiguousarray(np.asarray(offsets, dtype=np.int64))
    if off.ndim != 1 or off.shape[0] < 1:
        raise ValueError("offsets must be a 1-D array of rows+1 entries")
    if off[0] != 0 or np.any(np.diff(off) < 0):
        raise ValueError("offsets must start at 0 and never decrease")
    return off


def _ragged(name, x, offsets, nthreads, *extra_arrays, eps=None):
    x = _f64(x).reshape(-1)
    off = _offsets(offsets)
    rows = off.shape[0] - 1
    if off[-1] > x.shape[0]:
        raise ValueError("offsets run past the packed buffer")
    y = np.zeros_like(x)
    lib = _load()
    args = [_ptr(x), _ptr(y)] + [_ptr(a) for a in extra_arrays]
    args += [_ptr(off), rows]
    if eps is not None:
        args.append(_as_eps(eps))
    args.append(_threads(nthreads))
    getattr(lib, name)(*args)
    return y


def _max_len(off):
    return int(np.max(np.diff(off))) if off.shape[0] > 1 else 0


def softmax_ragged(x, offsets, nthreads=1):
    return _ragged("oracle_softmax_ragged", x, offsets, nthreads)


def logsoftmax_ragged(x, offsets, nthreads=1):
    return _ragged("oracle_logsoftmax_ragged", x, offsets, nthreads)


def layernorm_ragged(x, offsets, gamma=None, beta=None, eps=1e-5, nthreads=1):
    off = _offsets(offsets)
    n = max(_max_len(off), 1)
    return _ragged("oracle_layernorm_ragged", x, off, nthreads,
                   _vec(gamma, n, 1.0), _vec(beta, n, 0.0), eps=eps)


def rmsnorm_ragged(x, offsets, gamma=None, eps=1e-6, nthreads=1):
    off = _offsets(offsets)
    n = max(_max_len(off), 1)
    return _ragged("oracle_rmsnorm_ragged", x, off, nthreads,
                   _vec(gamma, n, 1.0), eps=eps)


def bucket(length: int, esize: int) -> int:
    """Row-length dispatch rule: 0 SMALL (<= 4 KiB), 1 MEDIUM (<= 32 KiB),
    2 LARGE, by the row's byte size."""
    return int(_load().oracle_bucket(int(length), int(esize)))


__all__ = ["build", "softmax", "logsoftmax", "layernorm", "rmsnorm",
           "softmax_ragged", "logsoftmax_ragged", "layernorm_ragged",
           "rmsnorm_ragged", "bucket", "SMALL", "MEDIUM", "LARGE"]


# ---------------------------------------------------------------------------
# Hyena FFT-size padding and the MoE group score (pad_moe_oracle.c)
# ---------------------------------------------------------------------------
def pad_scale(x, fft_size: int, scale: float):
    """``y[r, c] = scale * x[r, c]`` for ``c < seqlen``, then zeros up to
    ``fft_size`` (§6).  ``scale`` is taken as the float32 value the GPU
    multiplies by, widened to double; the product of two float32 values is
    exact in double."""
    x = _f64(x)
    if x.ndim != 2:
        raise ValueError("pad_scale wants a 2-D rows x seqlen array")
    rows, seqlen = x.shape
    if fft_size < seqlen:
        raise ValueError("fft_size < seqlen")
    y = np.empty((rows, fft_size), dtype=np.float64)
    _load().oracle_pad_scale(_ptr(x), _ptr(y), rows, seqlen, fft_size,
                             float(np.float32(scale)))
    return y


def moe_group_top2(scores, group: int = 32):
    """``out[t, g] = max_{i != j} (v_i + v_j)`` over each group of ``group``
    consecutive scores of token ``t`` (§2.1), by brute force over the pairs."""
    v = _f64(scores)
    if v.ndim != 2 or v.shape[1] % group:
        raise ValueError("moe_group_top2 wants tokens x experts, experts a multiple of group")
    tokens, experts = v.shape
    out = np.empty((tokens, experts // group), dtype=np.float64)
    _load().oracle_moe_group_top2(_ptr(v), _ptr(out), tokens, experts, group)
    return out


# ---------------------------------------------------------------------------
# Fused residual add + norm
# ---------------------------------------------------------------------------
def residual_sum(x, r, dtype):
    """The residual stream after the add, ``s = x + r``, as stored: the sum
    (exact in double for float32 / bfloat16 / float16 inputs but in
    pathological exponent gaps) rounded to nearest even in the I/O type
    ``dtype`` (a torch dtype), returned as float64."""
    import torch
    s = _f64(x) + _f64(r)
    return torch.from_numpy(s).to(dtype).double().numpy()


def add_layernorm(x, r, dtype, gamma=None, beta=None, eps=1e-5, nthreads=1):
    """``s = x + r`` stored in ``dtype``, then ``y = LayerNorm(s)``: the norm
    reads the sum as stored.  Returns ``(s, y)``."""
    s = residual_sum(x, r, dtype)
    return s, layernorm(s, gamma, beta, eps, nthreads)


def add_rmsnorm(x, r, dtype, gamma=None, eps=1e-6, nthreads=1):
    """``s = x + r`` stored in ``dtype``, then ``y = RMSNorm(s)``."""
    s = residual_sum(x, r, dtype)
    return s, rmsnorm(s, gamma, eps, nthreads)


# ---------------------------------------------------------------------------
# Backward passes (backward_oracle.c): analytic derivatives of the forward
# definitions above for an upstream gradient dy
# ---------------------------------------------------------------------------
def _pair(a, b, what):
    a = _f64(a)
    b = _f64(b)
    if a.ndim != 2 or a.shape != b.shape:
        raise ValueError(f"{what} wants two 2-D arrays of the same shape")
    return a, b


def softmax_backward(y, dy, nthreads=1):
    """``dx = y * (dy - sum(dy * y))`` per row, ``y`` the softmax output."""
    y, dy = _pair(y, dy, "softmax_backward")
    dx = np.empty_like(y)
    _load().oracle_softmax_backward(_ptr(y), _ptr(dy), _ptr(dx), y.shape[0], y.shape[1],
                                    _threads(nthreads))
    return dx


def logsoftmax_backward(y, dy, nthreads=1):
    """``dx = dy - exp(y) * sum(dy)`` per row, ``y`` the log-softmax output."""
    y, dy = _pair(y, dy, "logsoftmax_backward")
    dx = np.empty_like(y)
    _load().oracle_logsoftmax_backward(_ptr(y), _ptr(dy), _ptr(dx), y.shape[0], y.shape[1],
                                       _threads(nthreads))
    return dx


def layernorm_backward(x, dy, gamma=None, eps=1e-5, nthreads=1):
    """LayerNorm backward from the input ``x`` (statistics recomputed as the
    forward forms them).  Returns ``(dx, dgamma, dbeta)``; ``dgamma`` and
    ``dbeta`` are column sums over all rows."""
    x, dy = _pair(x, dy, "layernorm_backward")
    rows, cols = x.shape
    g = _vec(gamma, cols, 1.0)
    dx = np.empty_like(x)
    dg = np.empty(cols, dtype=np.float64)
    db = np.empty(cols, dtype=np.float64)
    rc = _load().oracle_layernorm_backward(_ptr(x), _ptr(dy), _ptr(g), _ptr(dx), _ptr(dg),
                                           _ptr(db), rows, cols, _as_eps(eps), _threads(nthreads))
    if rc != 0:
        raise MemoryError("oracle_layernorm_backward could not allocate its row statistics")
    return dx, dg, db


def rmsnorm_backward(x, dy, gamma=None, eps=1e-6, nthreads=1):
    """RMSNorm backward from the input ``x``.  Returns ``(dx, dgamma)``."""
    x, dy = _pair(x, dy, "rmsnorm_backward")
    rows, cols = x.shape
    g = _vec(gamma, cols, 1.0)
    dx = np.empty_like(x)
    dg = np.empty(cols, dtype=np.float64)
    rc = _load().oracle_rmsnorm_backward(_ptr(x), _ptr(dy), _ptr(g), _ptr(dx), _ptr(dg),
                                         rows, cols, _as_eps(eps), _threads(nthreads))
    if rc != 0:
        raise MemoryError("oracle_rmsnorm_backward could not allocate its row statistics")
    return dx, dg


def _ragged_norm_backward(dense_fn, x, dy, offsets, gamma, eps, nacc, nthreads):
    """Row ``i`` of a ragged norm is the dense norm of ``x[off[i]:off[i+1]]``
    with ``gamma[:len]``: its dx is the dense backward of that one row, and
    the parameter gradients of column ``j`` add up, in row order, the rows
    longer than ``j``.  Returns ``dx`` (packed like ``x``) and the ``nacc``
    column sums, each of max_len entries."""
    x = _f64(x).reshape(-1)
    dy = _f64(dy).reshape(-1)
    off = _offsets(offsets)
    if x.shape != dy.shape or off[-1] > x.shape[0]:
        raise ValueError("x and dy must be packed buffers of the same size holding every row")
    n = _max_len(off)
    g = _vec(gamma, max(n, 1), 1.0)
    dx = np.zeros_like(x)
    sums = [np.zeros(n, dtype=np.float64) for _ in range(nacc)]
    for i in range(off.shape[0] - 1):
        a, b = int(off[i]), int(off[i + 1])
        if b == a:
            continue
        out = dense_fn(x[None, a:b], dy[None, a:b], g[:b - a], eps=eps, nthreads=nthreads)
        dx[a:b] = out[0][0]
        for s, part in zip(sums, out[1:]):
            s[:b - a] += part
    return (dx, *sums)


def layernorm_backward_ragged(x, dy, offsets, gamma=None, eps=1e-5, nthreads=1):
    """LayerNorm backward over ragged rows (gamma indexed by the column inside
    the row).  Returns ``(dx, dgamma, dbeta)``, the last two of max_len
    entries."""
    return _ragged_norm_backward(layernorm_backward, x, dy, offsets, gamma, eps, 2, nthreads)


def rmsnorm_backward_ragged(x, dy, offsets, gamma=None, eps=1e-6, nthreads=1):
    """RMSNorm backward over ragged rows.  Returns ``(dx, dgamma)``."""
    return _ragged_norm_backward(rmsnorm_backward, x, dy, offsets, gamma, eps, 1, nthreads)
