"""Pins for the CPU oracle: checks that tie it to the mathematics rather than
to itself.  Each ``pin_*`` function takes an oracle module (the real one, or a
deliberately broken copy in the mutation tests) and raises AssertionError when
the oracle disagrees with

* closed forms derived by hand (``tests/golden/hand_cases.json``),
* invariants that any correct implementation satisfies,
* an independent brute-force restatement using ``math.fsum``,
* PyTorch's float64 CPU routines (a library, used only here),
* the row-length dispatch thresholds stated in the library's interface.
"""
from __future__ import annotations

import json
import math
import os

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")

_EXPR_NAMES = {"ln": math.log, "exp": math.exp, "sqrt": math.sqrt,
               "inf": math.inf}


def _ev(s: str) -> float:
    return float(eval(s, {"__builtins__": {}}, _EXPR_NAMES))  # noqa: S307


def _close(a, b, rtol=1e-13, atol=1e-14):
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    assert a.shape == b.shape, (a.shape, b.shape)
    ok = np.isclose(a, b, rtol=rtol, atol=atol, equal_nan=True)
    if not ok.all():
        with np.errstate(invalid="ignore"):
            d = np.where(ok, 0.0, np.abs(np.nan_to_num(a - b, nan=np.inf)))
        raise AssertionError(f"max |diff| {d.max()}\n{a}\n{b}")


def _call(orc, op, x, gamma=None, beta=None, eps=0.0):
    if op == "softmax":
        return orc.softmax(x)
    if op == "logsoftmax":
        return orc.logsoftmax(x)
    if op == "layernorm":
        return orc.layernorm(x, gamma, beta, eps=eps)
    if op == "rmsnorm":
        return orc.rmsnorm(x, gamma, eps=eps)
    raise ValueError(op)


def _call_ragged(orc, op, x, off, gamma=None, beta=None, eps=0.0):
    if op == "softmax":
        return orc.softmax_ragged(x, off)
    if op == "logsoftmax":
        return orc.logsoftmax_ragged(x, off)
    if op == "layernorm":
        return orc.layernorm_ragged(x, off, gamma, beta, eps=eps)
    if op == "rmsnorm":
        return orc.rmsnorm_ragged(x, off, gamma, eps=eps)
    raise ValueError(op)


OPS = ("softmax", "logsoftmax", "layernorm", "rmsnorm")


# --------------------------------------------------------------------------
def pin_hand_cases(orc):
    with open(os.path.join(GOLDEN, "hand_cases.json")) as f:
        cases = json.load(f)["cases"]
    for c in cases:
        x = np.array([[_ev(v) for v in row] for row in c["x"]])
        exp = np.array([[_ev(v) for v in row] for row in c["expected"]])
        g = np.array([_ev(v) for v in c["gamma"]]) if "gamma" in c else None
        b = np.array([_ev(v) for v in c["beta"]]) if "beta" in c else None
        got = _call(orc, c["op"], x, g, b, c.get("eps", 0.0))
        _close(got, exp, rtol=1e-14, atol=1e-15)
        # The same rows as a ragged batch give the same answer.
        off = np.arange(0, x.size + 1, x.shape[1], dtype=np.int64)
        got_r = _call_ragged(orc, c["op"], x.reshape(-1), off, g, b,
                             c.get("eps", 0.0))
        _close(got_r.reshape(x.shape), exp, rtol=1e-14, atol=1e-15)


def pin_softmax_invariants(orc):
    rng = np.random.default_rng(11)
    x = rng.normal(0, 4, size=(17, 61))
    p = orc.softmax(x)
    _close(p.sum(axis=1), np.ones(17), rtol=0, atol=1e-13)
    assert (p > 0).all() and (p < 1).all()
    # Order is preserved: argmax of softmax is argmax of x.
    assert (p.argmax(axis=1) == x.argmax(axis=1)).all()
    # Shift invariance.
    _close(orc.softmax(x + 123.25), p, rtol=1e-12, atol=1e-16)
    # log(softmax) == log-softmax, and log-softmax is shift invariant.
    ls = orc.logsoftmax(x)
    _close(np.log(p), ls, rtol=1e-12, atol=1e-13)
    _close(orc.logsoftmax(x - 77.5), ls, rtol=1e-12, atol=1e-12)
    # Ratios: p_i / p_j = exp(x_i - x_j).
    _close(p[:, 3] / p[:, 5], np.exp(x[:, 3] - x[:, 5]), rtol=1e-12)
    # Large entries (the long-row workload's +-80 spikes) do not overflow.
    z = np.zeros((1, 9))
    z[0, 2] = 80.0
    z[0, 7] = -80.0
    q = orc.softmax(z)
    assert np.isfinite(q).all()
    _close(q[0, 2], 1.0 / (1.0 + 7.0 * math.exp(-80.0) + math.exp(-160.0)),
           rtol=1e-14)


def pin_layernorm_invariants(orc):
    rng = np.random.default_rng(12)
    x = rng.normal(3, 2, size=(9, 47))
    y = orc.layernorm(x, eps=0.0)
    _close(y.mean(axis=1), np.zeros(9), rtol=0, atol=1e-13)
    _close(y.var(axis=1), np.ones(9), rtol=1e-12)
    # Affine invariance at eps = 0: LN(a x + b) == LN(x) for a > 0, and a
    # negative scale flips the sign.
    _close(orc.layernorm(2.5 * x - 40.0, eps=0.0), y, rtol=1e-10, atol=1e-12)
    _close(orc.layernorm(-0.5 * x, eps=0.0), -y, rtol=1e-10, atol=1e-12)
    # With eps > 0 the output variance is var/(var + eps).
    eps = 0.75
    ye = orc.layernorm(x, eps=eps)
    v = x.var(axis=1)
    _close(ye.var(axis=1), v / (v + np.float64(np.float32(eps))), rtol=1e-12)
    _close(ye.mean(axis=1), np.zeros(9), rtol=0, atol=1e-13)
    # Two distinct values normalise to -1, +1.
    _close(orc.layernorm(np.array([[4.0, 10.0]]), eps=0.0), [[-1.0, 1.0]])
    # gamma/beta act per column after normalising.
    g = rng.normal(1, 0.1, 47)
    b = rng.normal(0, 0.1, 47)
    _close(orc.layernorm(x, g, b, eps=0.0), y * g + b, rtol=1e-12, atol=1e-13)


def pin_rmsnorm_invariants(orc):
    rng = np.random.default_rng(13)
    x = rng.normal(0, 3, size=(8, 33))
    y = orc.rmsnorm(x, eps=0.0)
    # Unit root-mean-square at eps = 0, and scale invariance.
    _close(np.sqrt((y * y).mean(axis=1)), np.ones(8), rtol=1e-13)
    _close(orc.rmsnorm(17.0 * x, eps=0.0), y, rtol=1e-12)
    _close(orc.rmsnorm(-x, eps=0.0), -y, rtol=1e-12)
    # No mean subtraction: a constant row c gives c/sqrt(c^2 + eps) * gamma,
    # i.e. sign(c) * gamma at eps = 0.
    g = rng.normal(1, 0.1, 33)
    for c in (-2.5, 0.125, 9.0):
        row = np.full((1, 33), c)
        _close(orc.rmsnorm(row, g, eps=0.0), (np.sign(c) * g)[None],
               rtol=1e-14)
        eps = 0.5
        _close(orc.rmsnorm(row, g, eps=eps),
               (c / math.sqrt(c * c + eps) * g)[None], rtol=1e-14)
    # gamma acts per column.
    _close(orc.rmsnorm(x, g, eps=0.0), y * g, rtol=1e-12)


# --------------------------------------------------------------------------
def _brute_row(op, x, gamma, beta, eps):
    n = len(x)
    if op in ("softmax", "logsoftmax"):
        m = max(x)
        e = [math.exp(v - m) for v in x]
        s = math.fsum(e)
        if op == "softmax":
            return [v / s for v in e]
        return [(v - m) - math.log(s) for v in x]
    if op == "layernorm":
        mu = math.fsum(x) / n
        var = math.fsum([(v - mu) ** 2 for v in x]) / n
        d = math.sqrt(var + eps)
        return [(v - mu) / d * gamma[j] + beta[j] for j, v in enumerate(x)]
    if op == "rmsnorm":
        d = math.sqrt(math.fsum([v * v for v in x]) / n + eps)
        return [v / d * gamma[j] for j, v in enumerate(x)]
    raise ValueError(op)


def pin_brute_force(orc):
    rng = np.random.default_rng(14)
    for trial in range(40):
        rows = int(rng.integers(1, 9))
        cols = int(rng.integers(1, 34))
        op = OPS[trial % 4]
        x = rng.normal(0, 1 + trial % 5, size=(rows, cols))
        g = rng.normal(1, 0.2, cols)
        b = rng.normal(0, 0.2, cols)
        eps = float(np.float32([0.0, 1e-5, 1e-6, 0.1][trial % 4]))
        got = _call(orc, op, x, g, b, eps)
        exp = np.array([_brute_row(op, list(r), g, b, eps) for r in x])
        _close(got, exp, rtol=1e-11, atol=1e-12)


def pin_torch_float64(orc):
    import torch
    import torch.nn.functional as F
    rng = np.random.default_rng(15)
    x = rng.normal(0, 4, size=(6, 130))
    g = rng.normal(1, 0.1, 130)
    b = rng.normal(0, 0.1, 130)
    t = torch.from_numpy(x)
    _close(orc.softmax(x), torch.softmax(t, dim=1).numpy(), rtol=1e-12,
           atol=1e-15)
    _close(orc.logsoftmax(x), torch.log_softmax(t, dim=1).numpy(),
           rtol=1e-12, atol=1e-13)
    eps = float(np.float32(1e-5))
    _close(orc.layernorm(x, g, b, eps=eps),
           F.layer_norm(t, (130,), torch.from_numpy(g), torch.from_numpy(b),
                        eps=eps).numpy(), rtol=1e-11, atol=1e-12)
    if hasattr(F, "rms_norm"):
        eps = float(np.float32(1e-6))
        _close(orc.rmsnorm(x, g, eps=eps),
               F.rms_norm(t, (130,), torch.from_numpy(g), eps=eps).numpy(),
               rtol=1e-11, atol=1e-12)


def pin_ragged(orc):
    rng = np.random.default_rng(16)
    lens = np.array([5, 0, 1, 33, 2, 0, 17], dtype=np.int64)
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    x = rng.normal(0, 2, int(off[-1]))
    g = rng.normal(1, 0.1, int(lens.max()))
    b = rng.normal(0, 0.1, int(lens.max()))
    for op in OPS:
        eps = 1e-5 if op in ("layernorm", "rmsnorm") else 0.0
        y = _call_ragged(orc, op, x, off, g, b, eps)
        for i, n in enumerate(lens):
            seg = slice(off[i], off[i + 1])
            if n == 0:
                continue
            ref = _call(orc, op, x[seg][None, :], g[:n], b[:n], eps)[0]
            _close(y[seg], ref, rtol=0, atol=0)
        # gamma/beta are indexed by the column inside the row: a row of 2
        # sees gamma[0:2], not gamma[off:off+2].
    # Length-1 rows.
    one = np.arange(0, 4, dtype=np.int64)
    xs = np.array([3.0, -2.0, 0.5])
    _close(orc.softmax_ragged(xs, one), np.ones(3))
    _close(orc.logsoftmax_ragged(xs, one), np.zeros(3))
    _close(orc.layernorm_ragged(xs, one, np.array([2.0]), np.array([0.5]),
                                eps=1e-5), np.full(3, 0.5))


def pin_bucket_rule(orc):
    # Thresholds by row bytes: <= 4096 SMALL, <= 32768 MEDIUM, else LARGE.
    for esize in (2, 4):
        s_max = 4096 // esize
        m_max = 32768 // esize
        assert orc.bucket(1, esize) == 0
        assert orc.bucket(s_max, esize) == 0
        assert orc.bucket(s_max + 1, esize) == 1
        assert orc.bucket(m_max, esize) == 1
        assert orc.bucket(m_max + 1, esize) == 2
        assert orc.bucket(1 << 20, esize) == 2


def pin_pad_scale(orc):
    """Hyena FFT-size padding (§6): a hand-worked case, the zero tail, the
    identity at scale 1, linearity in the scale and row independence."""
    x = np.array([[1.0, 2.0, 3.0], [4.0, 5.0, 6.0]])
    want = np.array([[0.5, 1.0, 1.5, 0.0, 0.0], [2.0, 2.5, 3.0, 0.0, 0.0]])
    _close(orc.pad_scale(x, 5, 0.5), want, rtol=0, atol=0)
    g = np.random.default_rng(11)
    x = g.standard_normal((7, 13)).astype(np.float32).astype(np.float64)
    y = orc.pad_scale(x, 32, 0.25)
    assert y.shape == (7, 32)
    assert (y[:, 13:] == 0).all()
    _close(orc.pad_scale(x, 13, 1.0), x, rtol=0, atol=0)
    _close(orc.pad_scale(x, 20, 0.75), orc.pad_scale(x, 20, 0.5) + orc.pad_scale(x, 20, 0.25))
    perm = g.permutation(7)
    _close(orc.pad_scale(x[perm], 20, 0.5), orc.pad_scale(x, 20, 0.5)[perm], rtol=0, atol=0)
    # every live element is the scaled input element at the same position
    for r, c in ((0, 0), (3, 7), (6, 12)):
        assert y[r, c] == 0.25 * x[r, c]


def pin_moe_group_top2(orc):
    """MoE group score (§2.1): hand cases with ties and masked experts, the
    paper's statement that the largest off-diagonal pair sum is the sum of
    the two largest values (checked by sorting), invariance under permuting a
    group, and a shift by c moving the score by 2c."""
    inf = np.inf
    cases = [([5.0, 5.0, 1.0, 2.0], 10.0), ([1.0, 2.0, 3.0, 4.0], 7.0),
             ([-inf, 3.0, -inf, -inf], -inf), ([3.0, -1.0, -2.0, -5.0], 2.0),
             ([-inf, -inf, -inf, -inf], -inf), ([0.5, 0.5, 0.5, 0.5], 1.0)]
    for v, want in cases:
        got = orc.moe_group_top2(np.array([v]), group=4)
        assert got.shape == (1, 1)
        assert got[0, 0] == want, (v, got, want)
    g = np.random.default_rng(12)
    # coarse values so that ties, including tied maxima, are frequent
    v = np.round(g.standard_normal((50, 256)) * 4) / 4
    v[3, 40:72] = 1.0
    v[7, :32] = -inf
    v[7, 5] = 2.0
    got = orc.moe_group_top2(v)
    assert got.shape == (50, 8)
    top2 = np.sort(v.reshape(50, 8, 32), axis=2)[:, :, -2:].sum(axis=2)
    _close(got, top2, rtol=0, atol=0)
    assert got[3, 1] == 2.0 or got[3, 1] >= 2.0
    assert got[7, 0] == -inf
    perm = g.permutation(32)
    w = v.reshape(50, 8, 32)[:, :, perm].reshape(50, 256)
    _close(orc.moe_group_top2(w), got, rtol=0, atol=0)
    _close(orc.moe_group_top2(v + 1.5), got + 3.0, rtol=0, atol=0)


def pin_residual_norm(orc):
    """Fused residual add + norm: the stored sum of small integers is exact,
    a zero residual gives the plain norm of x, x and r commute, the sum is
    rounded to the I/O type before the norm reads it (a bf16 hand case), and
    the norms of the sum keep their invariants (mean 0 / unit RMS)."""
    import torch
    x = np.array([[1.0, 2.0, 3.0, 4.0], [-8.0, 0.0, 8.0, 16.0]])
    r = np.array([[10.0, 20.0, 30.0, 40.0], [1.0, 1.0, 1.0, 1.0]])
    s, y = orc.add_layernorm(x, r, torch.float32, eps=0.0)
    _close(s, [[11.0, 22.0, 33.0, 44.0], [-7.0, 1.0, 9.0, 17.0]], rtol=0, atol=0)
    # row 0 of s is 11 * (1, 2, 3, 4): mean 27.5, biased var 151.25
    _close(y[0], (np.array([11.0, 22.0, 33.0, 44.0]) - 27.5) / math.sqrt(151.25))
    # 256 + 1 is not a bf16 value: the sum rounds to 256 (ties to even) first
    s, _ = orc.add_rmsnorm(np.array([[256.0, 3.0]]), np.array([[1.0, 0.0]]), torch.bfloat16)
    _close(s, [[256.0, 3.0]], rtol=0, atol=0)
    g = np.random.default_rng(13)
    xv = g.standard_normal((6, 50)).astype(np.float32).astype(np.float64)
    rv = g.standard_normal((6, 50)).astype(np.float32).astype(np.float64)
    zero = np.zeros_like(xv)
    _close(orc.add_layernorm(xv, zero, torch.float32)[1], orc.layernorm(xv))
    _close(orc.add_rmsnorm(xv, zero, torch.float32)[1], orc.rmsnorm(xv))
    _close(orc.add_layernorm(xv, rv, torch.float32)[1], orc.add_layernorm(rv, xv, torch.float32)[1])
    s, y = orc.add_layernorm(xv, rv, torch.bfloat16, eps=0.0)
    assert (torch.from_numpy(s).to(torch.bfloat16).double().numpy() == s).all()
    _close(y.mean(axis=1), np.zeros(6), atol=1e-13)
    s, y = orc.add_rmsnorm(xv, rv, torch.float16, eps=0.0)
    _close(np.sqrt((y * y).mean(axis=1)), np.ones(6))


# --------------------------------------------------------------------------
# backward passes
# --------------------------------------------------------------------------
def _fd_grad(f, a, h=1e-5):
    """Central differences of the scalar function f at every entry of a."""
    a = np.array(a, dtype=np.float64)
    g = np.empty_like(a)
    flat = a.reshape(-1)
    gf = g.reshape(-1)
    for k in range(flat.size):
        old = flat[k]
        flat[k] = old + h
        fp = f(a)
        flat[k] = old - h
        fm = f(a)
        flat[k] = old
        gf[k] = (fp - fm) / (2 * h)
    return g


def pin_backward_finite_difference(orc):
    """Every backward pass against central differences of the (separately
    pinned) forward oracle: dx for all four operators, and dgamma / dbeta of
    the norms, of the loss sum(dy * f(x, gamma, beta))."""
    rng = np.random.default_rng(31)
    rows, n = 3, 9
    x = rng.normal(0.3, 2.0, (rows, n))
    dy = rng.normal(0.0, 1.0, (rows, n))
    g = rng.normal(1.0, 0.3, n)
    b = rng.normal(0.0, 0.3, n)
    tol = dict(rtol=1e-6, atol=1e-8)
    y = orc.softmax(x)
    _close(orc.softmax_backward(y, dy), _fd_grad(lambda a: np.sum(dy * orc.softmax(a)), x), **tol)
    y = orc.logsoftmax(x)
    _close(orc.logsoftmax_backward(y, dy),
           _fd_grad(lambda a: np.sum(dy * orc.logsoftmax(a)), x), **tol)
    eps = float(np.float32(1e-5))
    dx, dg, db = orc.layernorm_backward(x, dy, g, eps=eps)
    _close(dx, _fd_grad(lambda a: np.sum(dy * orc.layernorm(a, g, b, eps=eps)), x), **tol)
    _close(dg, _fd_grad(lambda a: np.sum(dy * orc.layernorm(x, a, b, eps=eps)), g), **tol)
    _close(db, _fd_grad(lambda a: np.sum(dy * orc.layernorm(x, g, a, eps=eps)), b), **tol)
    eps = float(np.float32(1e-6))
    dx, dg = orc.rmsnorm_backward(x, dy, g, eps=eps)
    _close(dx, _fd_grad(lambda a: np.sum(dy * orc.rmsnorm(a, g, eps=eps)), x), **tol)
    _close(dg, _fd_grad(lambda a: np.sum(dy * orc.rmsnorm(x, a, eps=eps)), g), **tol)


def pin_backward_ragged_norms(orc):
    """The ragged norm backward passes against central differences of the
    (separately pinned) ragged forward oracle, on rows of lengths 4, 0, 7, 1
    and 5 (an empty row, a one-element row, gamma columns reached by some rows
    only): dx, and dgamma / dbeta of max_len entries, of the loss
    sum(dy * f(x, gamma, beta)); then rows of one length, which must agree
    with the dense backward."""
    rng = np.random.default_rng(33)
    lens = np.array([4, 0, 7, 1, 5])
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    total, n = int(off[-1]), int(lens.max())
    x = rng.normal(0.4, 1.5, total)
    dy = rng.normal(0.0, 1.0, total)
    g = rng.normal(1.0, 0.3, n)
    b = rng.normal(0.0, 0.3, n)
    tol = dict(rtol=1e-6, atol=1e-8)
    eps = float(np.float32(1e-5))
    dx, dg, db = orc.layernorm_backward_ragged(x, dy, off, g, eps=eps)
    ln = lambda xx, gg, bb: np.sum(dy * orc.layernorm_ragged(xx, off, gg, bb, eps=eps))  # noqa: E731
    _close(dx, _fd_grad(lambda a: ln(a, g, b), x), **tol)
    _close(dg, _fd_grad(lambda a: ln(x, a, b), g), **tol)
    _close(db, _fd_grad(lambda a: ln(x, g, a), b), **tol)
    eps = float(np.float32(1e-6))
    dx, dg = orc.rmsnorm_backward_ragged(x, dy, off, g, eps=eps)
    rms = lambda xx, gg: np.sum(dy * orc.rmsnorm_ragged(xx, off, gg, eps=eps))  # noqa: E731
    _close(dx, _fd_grad(lambda a: rms(a, g), x), **tol)
    _close(dg, _fd_grad(lambda a: rms(x, a), g), **tol)
    # equal lengths: the dense backward of the same rows
    xe = rng.normal(0.0, 2.0, (3, 6))
    de = rng.normal(0.0, 1.0, (3, 6))
    ge = rng.normal(1.0, 0.3, 6)
    offe = np.arange(0, 19, 6, dtype=np.int64)
    for got, exp in zip(orc.layernorm_backward_ragged(xe.reshape(-1), de.reshape(-1), offe, ge),
                        orc.layernorm_backward(xe, de, ge)):
        _close(got, exp.reshape(-1), rtol=1e-14, atol=1e-15)


def pin_backward_invariants(orc):
    """Properties any correct backward pass has: softmax-family gradients sum
    to zero over a row; a constant upstream gradient gives no softmax
    gradient; the log-softmax gradient of one log-probability is e_k - p;
    the two-element softmax closed form; LayerNorm gradients are orthogonal
    to 1 and to xhat (eps = 0), vanish for two-element rows (eps = 0) and are
    unchanged by a shift of x; RMSNorm gradients are orthogonal to x and
    scale as 1/c when x does (eps = 0); dbeta is the column sum of dy."""
    rng = np.random.default_rng(32)
    x = rng.normal(0.0, 2.0, (5, 17))
    dy = rng.normal(0.0, 1.0, (5, 17))
    g = rng.normal(1.0, 0.3, 17)
    p = orc.softmax(x)
    _close(orc.softmax_backward(p, dy).sum(axis=1), np.zeros(5), atol=1e-14)
    _close(orc.softmax_backward(p, np.full_like(x, 0.7)), np.zeros_like(x), atol=1e-15)
    lp = orc.logsoftmax(x)
    _close(orc.logsoftmax_backward(lp, dy).sum(axis=1), np.zeros(5), atol=1e-13)
    onehot = np.zeros_like(x)
    onehot[np.arange(5), [0, 3, 16, 8, 8]] = 1.0
    _close(orc.logsoftmax_backward(lp, onehot), onehot - p, rtol=1e-13, atol=1e-15)
    # two elements: y1 = 1 / (1 + exp(x2 - x1)); dx1 = y1 y2 (dy1 - dy2) = -dx2
    x2 = np.array([[0.5, -1.25]])
    d2 = np.array([[2.0, -0.5]])
    s1 = 1.0 / (1.0 + math.exp(-1.75))
    want = s1 * (1.0 - s1) * 2.5
    _close(orc.softmax_backward(orc.softmax(x2), d2), [[want, -want]], rtol=1e-14)
    # LayerNorm, eps = 0
    dx, dg, db = orc.layernorm_backward(x, dy, g, eps=0.0)
    mu = x.mean(axis=1, keepdims=True)
    xhat = (x - mu) / np.sqrt(((x - mu) ** 2).mean(axis=1, keepdims=True))
    _close(dx.sum(axis=1), np.zeros(5), atol=1e-13)
    _close((dx * xhat).sum(axis=1), np.zeros(5), atol=1e-13)
    _close(db, dy.sum(axis=0), rtol=1e-15, atol=1e-15)
    _close(orc.layernorm_backward(x + 3.5, dy, g, eps=1e-3)[0],
           orc.layernorm_backward(x, dy, g, eps=1e-3)[0], rtol=1e-9, atol=1e-12)
    _close(orc.layernorm_backward(2.0 * x, dy, g, eps=0.0)[0], dx / 2.0, rtol=1e-12, atol=1e-14)
    _close(orc.layernorm_backward(x[:, :2], dy[:, :2], g[:2], eps=0.0)[0], np.zeros((5, 2)),
           atol=1e-14)
    # RMSNorm, eps = 0
    dx, dg = orc.rmsnorm_backward(x, dy, g, eps=0.0)
    _close((dx * x).sum(axis=1), np.zeros(5), atol=1e-13)
    _close(orc.rmsnorm_backward(4.0 * x, dy, g, eps=0.0)[0], dx / 4.0, rtol=1e-12, atol=1e-14)
    _close(orc.rmsnorm_backward(4.0 * x, dy, g, eps=0.0)[1], dg, rtol=1e-12, atol=1e-14)
    # one-element rows: LayerNorm's output is beta whatever x is
    _close(orc.layernorm_backward(x[:, :1], dy[:, :1], g[:1], eps=1e-5)[0], np.zeros((5, 1)),
           atol=0)


def pin_backward_torch(orc):
    """Against PyTorch autograd in float64 (a library, used only here),
    including dgamma / dbeta summed over many rows."""
    import torch
    import torch.nn.functional as F
    rng = np.random.default_rng(33)
    x = rng.normal(0.5, 3.0, (40, 130))
    dy = rng.normal(0.0, 1.0, (40, 130))
    gam = rng.normal(1.0, 0.2, 130)
    bet = rng.normal(0.0, 0.2, 130)
    td = torch.from_numpy(dy)

    def grads(fn, *args):
        ts = [torch.from_numpy(a.copy()).requires_grad_(True) for a in args]
        (fn(*ts) * td).sum().backward()
        return [t.grad.numpy() for t in ts]

    t = torch.from_numpy(x)
    y = torch.softmax(t, dim=1).numpy()
    _close(orc.softmax_backward(y, dy), grads(lambda a: torch.softmax(a, dim=1), x)[0],
           rtol=1e-11, atol=1e-14)
    y = torch.log_softmax(t, dim=1).numpy()
    _close(orc.logsoftmax_backward(y, dy), grads(lambda a: torch.log_softmax(a, dim=1), x)[0],
           rtol=1e-11, atol=1e-13)
    eps = float(np.float32(1e-5))
    dx, dg, db = orc.layernorm_backward(x, dy, gam, eps=eps)
    want = grads(lambda a, g_, b_: F.layer_norm(a, (130,), g_, b_, eps=eps), x, gam, bet)
    _close(dx, want[0], rtol=1e-10, atol=1e-12)
    _close(dg, want[1], rtol=1e-10, atol=1e-11)
    _close(db, want[2], rtol=1e-10, atol=1e-11)
    if hasattr(F, "rms_norm"):
        eps = float(np.float32(1e-6))
        dx, dg = orc.rmsnorm_backward(x, dy, gam, eps=eps)
        want = grads(lambda a, g_: F.rms_norm(a, (130,), g_, eps=eps), x, gam)
        _close(dx, want[0], rtol=1e-10, atol=1e-12)
        _close(dg, want[1], rtol=1e-10, atol=1e-11)


ALL_PINS = [pin_hand_cases, pin_softmax_invariants, pin_layernorm_invariants,
            pin_rmsnorm_invariants, pin_brute_force, pin_torch_float64,
            pin_ragged, pin_bucket_rule, pin_pad_scale, pin_moe_group_top2,
            pin_residual_norm, pin_backward_finite_difference, pin_backward_invariants,
            pin_backward_torch, pin_backward_ragged_norms]
