"""Randomised parity sweep through the C ABI: seeded random shapes, row
strides, element offsets (16-byte congruent or not), dtypes, in-place calls
and operators -- forward (dense and ragged, with a first offset other than 0)
and the backward passes, dense and ragged -- each checked against the double-precision oracle
with the tolerance its own tests use.  Every case is a pure function of its seed, so a
failure names a reproducible case."""
import numpy as np
import pytest
import torch

from oracle import rowop_oracle as orc
from tests.gpu_util import (DTYPES, ESIZE, assert_close, canary_tensor, eps_for, is_canary,
                            oracle_dense, oracle_ragged, to_f64)
from tests.test_gpu_backward import R_COMP, R_COMP_PARAM, check, oracle as bwd_oracle, scales

pytestmark = pytest.mark.gpu
G = 64
FWD = ("softmax", "logsoftmax", "layernorm", "rmsnorm")


@pytest.fixture(scope="module")
def rw():
    from paper_2607_23089_gb300 import build, rowop
    build.build()
    rowop.load()
    torch.cuda.set_device(0)
    return rowop


def _shape(g, max_elems=1_500_000):
    """rows, cols, ld: cols log-uniform over 1..80000, the product bounded."""
    cols = int(np.exp(g.uniform(0, np.log(80000))))
    cols = max(1, cols)
    rows = int(g.integers(1, max(2, min(40, max_elems // cols)) + 1))
    ld = cols + int(g.choice([0, 0, 1, 3, 8, 17]))
    return rows, cols, ld


def _buf(g, rows, ld, dtype, fill=None):
    off = int(g.integers(0, 8))
    b = canary_tensor(G + off + rows * ld + G, dtype)
    if fill is not None:
        b[G + off:G + off + rows * ld] = fill.reshape(-1).cuda()
    return b, G + off


def _ptr(b, o, dtype):
    return b.data_ptr() + o * ESIZE[dtype]


def fwd_case(rw, seed):
    g = np.random.default_rng(seed)
    op = FWD[seed % 4]
    dtype = DTYPES[(seed // 4) % 3]
    rows, cols, ld = _shape(g)
    tg = torch.Generator("cpu").manual_seed(seed)
    x = (float(g.uniform(0.5, 6)) * torch.randn(rows, ld, generator=tg) +
         float(g.uniform(-2, 2))).to(dtype)
    xb, xo = _buf(g, rows, ld, dtype, x)
    inplace = g.random() < 0.2
    yb, yo = (xb, xo) if inplace else _buf(g, rows, ld, dtype)
    gam = bet = None
    if op in ("layernorm", "rmsnorm") and g.random() < 0.8:
        gam = (1 + 0.2 * torch.randn(cols, generator=tg)).to(dtype)
        bet = (0.2 * torch.randn(cols, generator=tg)).to(dtype) if op == "layernorm" else None
    eps = eps_for(op)
    code = rw.dtype_code(dtype)
    s = torch.cuda.current_stream().cuda_stream
    gp = gam.cuda() if gam is not None else None
    bp = bet.cuda() if bet is not None else None
    a, o = _ptr(xb, xo, dtype), _ptr(yb, yo, dtype)
    if op == "softmax":
        st = rw.rowop_softmax(a, o, rows, cols, ld, code, s)
    elif op == "logsoftmax":
        st = rw.rowop_logsoftmax(a, o, rows, cols, ld, code, s)
    elif op == "layernorm":
        st = rw.rowop_layernorm(a, o, gp.data_ptr() if gp is not None else None,
                                bp.data_ptr() if bp is not None else None, rows, cols, ld, code,
                                eps, s)
    else:
        st = rw.rowop_rmsnorm(a, o, gp.data_ptr() if gp is not None else None, rows, cols, ld,
                              code, eps, s)
    assert st == 0, (seed, rw.STATUS.get(st, st))
    assert rw.check_status() == 0
    y = yb[yo:yo + rows * ld].view(rows, ld)
    ref = oracle_dense(op, x[:, :cols].double().numpy(),
                       None if gam is None else gam.double().numpy(),
                       None if bet is None else bet.double().numpy(), eps)
    assert_close(to_f64(y[:, :cols]), ref, dtype, f"seed {seed}: {op} {dtype} {rows}x{cols} ld {ld}")
    assert is_canary(yb[:yo]).all() and is_canary(yb[yo + rows * ld:]).all()
    if ld > cols and not inplace:
        assert is_canary(y[:, cols:]).all()


def ragged_case(rw, seed):
    g = np.random.default_rng(10_000 + seed)
    op = FWD[seed % 4]
    dtype = DTYPES[(seed // 4) % 3]
    rows = int(g.integers(1, 60))
    max_len = int(np.exp(g.uniform(0, np.log(70000))))
    lens = np.minimum(max_len, np.exp(g.uniform(0, np.log(max_len + 1), rows)).astype(np.int64))
    lens[g.random(rows) < 0.1] = 0
    start = int(g.integers(0, 9))
    off = (start + np.concatenate([[0], np.cumsum(lens)])).astype(np.int64)
    total = int(off[-1])
    tg = torch.Generator("cpu").manual_seed(seed)
    x = (3 * torch.randn(max(total, 1), generator=tg)).to(dtype)
    xb, xo = _buf(g, 1, max(total, 1), dtype, x)
    yb, yo = _buf(g, 1, max(total, 1), dtype)
    gam = (1 + 0.1 * torch.randn(max(max_len, 1), generator=tg)).to(dtype)
    bet = (0.1 * torch.randn(max(max_len, 1), generator=tg)).to(dtype)
    eps = eps_for(op)
    offd = torch.from_numpy(off).cuda()
    ws = rw.ragged_workspace(rows)
    code = rw.dtype_code(dtype)
    s = torch.cuda.current_stream().cuda_stream
    a, o = _ptr(xb, xo, dtype), _ptr(yb, yo, dtype)
    gd, bd = gam.cuda(), bet.cuda()
    if op == "softmax":
        st = rw.rowop_softmax_ragged(a, o, offd.data_ptr(), rows, max_len, code, ws.data_ptr(),
                                     ws.numel(), s)
    elif op == "logsoftmax":
        st = rw.rowop_logsoftmax_ragged(a, o, offd.data_ptr(), rows, max_len, code,
                                        ws.data_ptr(), ws.numel(), s)
    elif op == "layernorm":
        st = rw.rowop_layernorm_ragged(a, o, gd.data_ptr(), bd.data_ptr(), offd.data_ptr(), rows,
                                       max_len, code, eps, ws.data_ptr(), ws.numel(), s)
    else:
        st = rw.rowop_rmsnorm_ragged(a, o, gd.data_ptr(), offd.data_ptr(), rows, max_len, code,
                                     eps, ws.data_ptr(), ws.numel(), s)
    assert st == 0, (seed, rw.STATUS.get(st, st))
    assert rw.check_status() == 0
    if total > start:
        y = to_f64(yb[yo + start:yo + total])
        ref = oracle_ragged(op, x[start:total].double().numpy(), off - start,
                            gam.double().numpy(), bet.double().numpy(), eps)
        assert_close(y, ref, dtype, f"seed {seed}: ragged {op} {dtype} rows {rows} max_len {max_len}")
    assert is_canary(yb[:yo + start]).all() and is_canary(yb[yo + total:]).all()


def bwd_case(rw, seed):
    g = np.random.default_rng(20_000 + seed)
    op = FWD[seed % 4]
    dtype = DTYPES[(seed // 4) % 3]
    rows, cols, ld = _shape(g, 1_000_000)
    tg = torch.Generator("cpu").manual_seed(seed)
    if op in ("softmax", "logsoftmax"):
        x = (3.0 * torch.randn(rows, cols, generator=tg, dtype=torch.float64)).numpy()
        a = torch.from_numpy(orc.softmax(x) if op == "softmax" else orc.logsoftmax(x)).to(dtype)
    else:
        a = (2.0 * torch.randn(rows, cols, generator=tg) + 0.3).to(dtype)
    dy = torch.randn(rows, cols, generator=tg).to(dtype)
    gam = (1 + 0.2 * torch.randn(cols, generator=tg)).to(dtype) if op in ("layernorm", "rmsnorm") else None
    pad = lambda t: torch.nn.functional.pad(t.float(), (0, ld - cols)).to(dtype)  # noqa: E731
    ab, ao = _buf(g, rows, ld, dtype, pad(a))
    db, do = _buf(g, rows, ld, dtype, pad(dy))
    xb, xo = _buf(g, rows, ld, dtype)
    eps = eps_for(op)
    code = rw.dtype_code(dtype)
    s = torch.cuda.current_stream().cuda_stream
    p = lambda b, o: _ptr(b, o, dtype)  # noqa: E731
    dg = torch.empty(cols, dtype=dtype, device="cuda")
    dbt = torch.empty(cols, dtype=dtype, device="cuda")
    if op == "softmax":
        st = rw.rowop_softmax_backward(p(ab, ao), p(db, do), p(xb, xo), rows, cols, ld, code, s)
    elif op == "logsoftmax":
        st = rw.rowop_logsoftmax_backward(p(ab, ao), p(db, do), p(xb, xo), rows, cols, ld, code, s)
    else:
        size = (rw.rowop_layernorm_backward_workspace_size(cols) if op == "layernorm"
                else rw.rowop_rmsnorm_backward_workspace_size(cols))
        ws = torch.empty(size, dtype=torch.uint8, device="cuda")
        if op == "layernorm":
            st = rw.rowop_layernorm_backward(p(ab, ao), p(db, do), gam.cuda().data_ptr(), p(xb, xo),
                                             dg.data_ptr(), dbt.data_ptr(), rows, cols, ld, code,
                                             eps, ws.data_ptr(), ws.numel(), s)
        else:
            st = rw.rowop_rmsnorm_backward(p(ab, ao), p(db, do), gam.cuda().data_ptr(), p(xb, xo),
                                           dg.data_ptr(), rows, cols, ld, code, eps,
                                           ws.data_ptr(), ws.numel(), s)
    assert st == 0, (seed, rw.STATUS.get(st, st))
    assert rw.check_status() == 0
    a64, dy64 = a.double().numpy(), dy.double().numpy()
    g64 = gam.double().numpy() if gam is not None else None
    f32eps = float(np.float32(eps))
    rdx, rdg, rdb = bwd_oracle(op, a64, dy64, g64, f32eps)
    sdx, sdg, sdb = scales(op, a64, dy64, g64, f32eps)
    what = f"seed {seed}: {op} backward {dtype} {rows}x{cols} ld {ld}"
    dx = xb[xo:xo + rows * ld].view(rows, ld)
    check(to_f64(dx[:, :cols]), rdx, sdx, dtype, R_COMP, what + " dx")
    if ld > cols:
        assert is_canary(dx[:, cols:]).all()
    if op in ("layernorm", "rmsnorm"):
        check(to_f64(dg), rdg, sdg, dtype, R_COMP_PARAM, what + " dgamma")
    if op == "layernorm":
        check(to_f64(dbt), rdb, sdb, dtype, R_COMP_PARAM, what + " dbeta")


def ragged_bwd_case(rw, seed):
    """Ragged LayerNorm / RMSNorm backward: random row count, lengths
    log-uniform up to 70000 (empty rows included), a random first offset,
    dtype, gamma present or not, which gradients are wanted, dx in place."""
    from tests.test_gpu_backward_ragged_norm import call, make_inputs, reference, verify
    g = np.random.default_rng(30_000 + seed)
    op = ("layernorm", "rmsnorm")[seed % 2]
    dtype = DTYPES[(seed // 2) % 3]
    rows = int(g.integers(1, 40))
    top = int(np.exp(g.uniform(0, np.log(70000))))
    lens = np.minimum(top, np.exp(g.uniform(0, np.log(top + 1), rows)).astype(np.int64))
    lens[g.random(rows) < 0.1] = 0
    max_len = int(lens.max()) + int(g.integers(0, 50))
    affine = g.random() < 0.8
    x, dy, gam, off = make_inputs(dtype, lens, max_len, seed=seed, base_off=int(g.integers(0, 9)),
                                  affine=affine)
    want = (bool(g.random() < 0.8), bool(g.random() < 0.8))
    inplace = (None, None, "dy", "x")[int(g.integers(0, 4))]
    st, dxb, dgb, dbb = call(rw, op, dtype, x, dy, gam, off, max_len, inplace, want)
    assert st == 0, (seed, rw.STATUS.get(st, st))
    assert rw.check_status() == 0
    dx_rows, params, ps = reference(op, x, dy, gam, off, max_len)
    verify(op, dtype, dx_rows, params, ps, off, dxb, dgb, dbb, max_len,
           f"seed {seed}: ragged {op} backward {dtype} rows {rows} max_len {max_len}")


BATCH = 12


@pytest.mark.parametrize("batch", range(30))
def test_fuzz_dense_forward(rw, batch):
    for seed in range(batch * BATCH, (batch + 1) * BATCH):
        fwd_case(rw, seed)


@pytest.mark.parametrize("batch", range(18))
def test_fuzz_ragged_forward(rw, batch):
    for seed in range(batch * BATCH, (batch + 1) * BATCH):
        ragged_case(rw, seed)


@pytest.mark.parametrize("batch", range(24))
def test_fuzz_backward(rw, batch):
    for seed in range(batch * BATCH, (batch + 1) * BATCH):
        bwd_case(rw, seed)


@pytest.mark.parametrize("batch", range(8))
def test_fuzz_ragged_norm_backward(rw, batch):
    for seed in range(batch * BATCH, (batch + 1) * BATCH):
        ragged_bwd_case(rw, seed)
