"""GPU parity of the backward passes (softmax, log-softmax, LayerNorm,
RMSNorm), through the C ABI, against the double-precision oracle.

Inputs: the softmax family takes the forward output y, made here by the
oracle's own forward on a seeded x and rounded to the I/O type (the GPU and
the oracle see the same y); the norms take a seeded x.  dy is seeded.

Tolerance, derived from the arithmetic (fp32 inside, the I/O type outside):
every output is a short fp32 expression of row sums, and the error of an fp32
sum of terms t_i is bounded by k * 2^-24 * sum |t_i| for k additions in a
chain (here a thread's slots, a butterfly, a warp / rank merge chain: k well
under 100).  So each output o is held to

    |o_gpu - o_ref| <= r_out * |o_ref| + r_comp * S(o) + a_out

with S(o) the sum of the magnitudes of the terms that make it up (computed
below in double from the inputs: a scale, not an expected value), r_comp =
1e-5 (fp32 arithmetic, k * 2^-24 < 1e-5), and r_out the output rounding:
1e-6 (fp32), 1e-2 (bf16, as for the forward operators), 1e-3 (fp16), and
a_out the absolute rounding step of fp16 subnormals, 2^-24 (1e-30 otherwise).
dgamma / dbeta sum over rows in per-CTA partials, then over the partials:
their chains are longer, r_comp = 3e-5 there.
"""
import numpy as np
import pytest
import torch

from oracle import rowop_oracle as orc
from tests.gpu_util import DTYPE_IDS, DTYPES, ESIZE, canary_tensor, is_canary, to_f64

pytestmark = pytest.mark.gpu

R_OUT = {torch.float32: 1e-6, torch.bfloat16: 1e-2, torch.float16: 1e-3}
# fp16 results below 2^-14 are subnormal: their rounding step is 2^-24
A_OUT = {torch.float32: 1e-30, torch.bfloat16: 1e-30, torch.float16: 2.0 ** -24}
R_COMP = 1e-5
R_COMP_PARAM = 3e-5
NORMS = ("layernorm", "rmsnorm")
OPS = ("softmax", "logsoftmax", "layernorm", "rmsnorm")
G = 64  # guard elements around every buffer


@pytest.fixture(scope="module")
def rw():
    from paper_2607_23089_gb300 import build, rowop
    build.build()
    rowop.load()
    torch.cuda.set_device(0)
    return rowop


def _bits(t):
    return t.view(torch.int32) if t.dtype == torch.float32 else t.view(torch.int16)


def check(got, ref, scale, dtype, r_comp, what):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape
    assert np.isfinite(got).all(), f"{what}: non-finite output"
    lim = R_OUT[dtype] * np.abs(ref) + r_comp * scale + A_OUT[dtype]
    err = np.abs(got - ref)
    bad = err > lim
    if bad.any():
        i = np.unravel_index(np.argmax(err - lim), err.shape)
        raise AssertionError(f"{what}: {int(bad.sum())} of {bad.size} out of tolerance; worst "
                             f"at {i}: got {got[i]!r} ref {ref[i]!r} err {err[i]:.3e} "
                             f"lim {lim[i]:.3e}")


def scales(op, a, dy, gam, eps):
    """Magnitude scales S of dx, dgamma, dbeta for the tolerance (double)."""
    n = a.shape[1]
    if op == "softmax":
        return np.abs(a) * (np.abs(dy) + np.abs(dy * a).sum(1, keepdims=True)), None, None
    if op == "logsoftmax":
        return np.abs(dy) + np.exp(a) * np.abs(dy).sum(1, keepdims=True), None, None
    g = dy * gam[None, :]
    if op == "layernorm":
        mu = a.mean(1, keepdims=True)
        rstd = 1.0 / np.sqrt(((a - mu) ** 2).mean(1, keepdims=True) + eps)
        xh = np.abs((a - mu) * rstd) + 1.0
    else:
        rstd = 1.0 / np.sqrt((a * a).mean(1, keepdims=True) + eps)
        xh = np.abs(a * rstd) + 1.0
    s_dx = rstd * (np.abs(g) + np.abs(g).sum(1, keepdims=True) / n
                   + xh * (np.abs(g) * xh).sum(1, keepdims=True) / n)
    return s_dx, (np.abs(dy) * xh).sum(0), np.abs(dy).sum(0)


def _place(t, ld, off, dtype):
    """A canary buffer holding the rows of t at row stride ld, offset off."""
    rows, cols = t.shape
    buf = canary_tensor(G + off + rows * ld + G, dtype)
    if rows:
        view = buf[G + off:G + off + rows * ld].view(rows, ld)
        view[:, :cols] = t.cuda()
    return buf, G + off


def inputs(op, dtype, rows, cols, seed, affine=True):
    g = torch.Generator("cpu").manual_seed(seed)
    if op in ("softmax", "logsoftmax"):
        x = (3.0 * torch.randn(rows, cols, generator=g, dtype=torch.float64)).numpy()
        y = orc.softmax(x) if op == "softmax" else orc.logsoftmax(x)
        a = torch.from_numpy(y).to(dtype)
    else:
        a = (2.0 * torch.randn(rows, cols, generator=g) + 0.3).to(dtype)
    dy = torch.randn(rows, cols, generator=g).to(dtype)
    gam = None
    if op in NORMS and affine:
        gam = (1.0 + 0.2 * torch.randn(cols, generator=g)).to(dtype)
    return a, dy, gam


def oracle(op, a64, dy64, g64, eps):
    if op == "softmax":
        return orc.softmax_backward(a64, dy64), None, None
    if op == "logsoftmax":
        return orc.logsoftmax_backward(a64, dy64), None, None
    if op == "layernorm":
        return orc.layernorm_backward(a64, dy64, g64, eps=eps)
    dx, dg = orc.rmsnorm_backward(a64, dy64, g64, eps=eps)
    return dx, dg, None


def run_bwd(rw, op, dtype, rows, cols, ld=None, offs=(0, 0, 0), inplace=None, seed=0,
            affine=True, want=(True, True), eps=None, compare=True):
    """One backward call on guarded buffers; checks the result against the
    oracle and that nothing outside the outputs was written.  Returns the
    device results (dx rows, dgamma, dbeta) for further checks."""
    ld = ld or cols
    es = ESIZE[dtype]
    eps = eps if eps is not None else (1e-5 if op == "layernorm" else 1e-6)
    a, dy, gam = inputs(op, dtype, rows, cols, seed, affine)
    ab, ao = _place(a, ld, offs[0], dtype)
    db_, do = _place(dy, ld, offs[1], dtype)
    if inplace == "dy":
        xb, xo = db_, do
    elif inplace == "a":
        xb, xo = ab, ao
    else:
        xb, xo = canary_tensor(G + offs[2] + rows * ld + G, dtype), G + offs[2]
    norm = op in NORMS
    want_g = norm and want[0]
    want_b = op == "layernorm" and want[1]
    dg_buf = canary_tensor(G + cols + G, dtype) if want_g else None
    dbt_buf = canary_tensor(G + cols + G, dtype) if want_b else None
    p = lambda b, o: b.data_ptr() + o * es  # noqa: E731
    gd = gam.cuda() if gam is not None else None
    s = torch.cuda.current_stream().cuda_stream
    code = rw.dtype_code(dtype)
    ws = None
    if want_g or want_b:
        size = (rw.rowop_layernorm_backward_workspace_size(cols) if op == "layernorm"
                else rw.rowop_rmsnorm_backward_workspace_size(cols))
        assert size > 0
        ws = torch.empty(size, dtype=torch.uint8, device="cuda")
    wp = ws.data_ptr() if ws is not None else None
    wn = ws.numel() if ws is not None else 0
    if op == "softmax":
        st = rw.rowop_softmax_backward(p(ab, ao), p(db_, do), p(xb, xo), rows, cols, ld, code, s)
    elif op == "logsoftmax":
        st = rw.rowop_logsoftmax_backward(p(ab, ao), p(db_, do), p(xb, xo), rows, cols, ld,
                                          code, s)
    elif op == "layernorm":
        st = rw.rowop_layernorm_backward(p(ab, ao), p(db_, do), gd.data_ptr() if gd is not None
                                         else None, p(xb, xo),
                                         p(dg_buf, G) if want_g else None,
                                         p(dbt_buf, G) if want_b else None, rows, cols, ld,
                                         code, eps, wp, wn, s)
    else:
        st = rw.rowop_rmsnorm_backward(p(ab, ao), p(db_, do), gd.data_ptr() if gd is not None
                                       else None, p(xb, xo),
                                       p(dg_buf, G) if want_g else None, rows, cols, ld, code,
                                       eps, wp, wn, s)
    assert st == 0, rw.STATUS.get(st, st)
    assert rw.check_status() == 0
    dx = xb[xo:xo + rows * ld].view(rows, ld) if rows else xb[:0].view(0, ld)
    # guards and ld gaps untouched
    assert is_canary(xb[:xo]).all() and is_canary(xb[xo + rows * ld:]).all()
    if ld > cols and inplace is None:
        assert is_canary(dx[:, cols:]).all()
    for buf in (dg_buf, dbt_buf):
        if buf is not None:
            assert is_canary(buf[:G]).all() and is_canary(buf[G + cols:]).all()
    dgam = dg_buf[G:G + cols] if want_g else None
    dbet = dbt_buf[G:G + cols] if want_b else None
    if compare:
        a64, dy64 = a.double().numpy(), dy.double().numpy()
        g64 = gam.double().numpy() if gam is not None else np.ones(cols)
        f32eps = float(np.float32(eps))
        ref_dx, ref_dg, ref_db = oracle(op, a64, dy64, g64, f32eps)
        s_dx, s_dg, s_db = scales(op, a64, dy64, g64, f32eps)
        if rows:
            check(to_f64(dx[:, :cols]), ref_dx, s_dx, dtype, R_COMP, f"{op} dx")
        if want_g:
            check(to_f64(dgam), ref_dg, s_dg, dtype, R_COMP_PARAM, f"{op} dgamma")
        if want_b:
            check(to_f64(dbet), ref_db, s_db, dtype, R_COMP_PARAM, f"{op} dbeta")
    return dx[:, :cols].clone(), dgam, dbet


COLS = [1, 7, 64, 100, 513, 1000, 2048, 3001, 4096, 6000, 8192, 12000, 20000, 40000]


@pytest.mark.parametrize("dtype", DTYPES, ids=DTYPE_IDS)
@pytest.mark.parametrize("op", OPS)
@pytest.mark.parametrize("cols", COLS)
def test_backward_parity(rw, op, dtype, cols):
    rows = 23 if cols <= 8192 else 5
    run_bwd(rw, op, dtype, rows, cols, seed=cols)


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16], ids=["f32", "bf16"])
@pytest.mark.parametrize("op,cols", [("softmax", 262144), ("logsoftmax", 131072),
                                     ("layernorm", 262144), ("rmsnorm", 65536),
                                     ("logsoftmax", 100003)])
def test_backward_long_rows(rw, op, dtype, cols):
    """Rows split over clusters, up to the longest row accepted."""
    run_bwd(rw, op, dtype, 3, cols, seed=cols + 1)


@pytest.mark.parametrize("op", OPS)
def test_backward_too_long(rw, op):
    cap = 262144
    x = torch.zeros(1, cap + 1, device="cuda")
    s = torch.cuda.current_stream().cuda_stream
    F32 = rw.ROWOP_F32
    if op == "softmax":
        st = rw.rowop_softmax_backward(x.data_ptr(), x.data_ptr(), x.data_ptr(), 1, cap + 1,
                                       cap + 1, F32, s)
    elif op == "logsoftmax":
        st = rw.rowop_logsoftmax_backward(x.data_ptr(), x.data_ptr(), x.data_ptr(), 1, cap + 1,
                                          cap + 1, F32, s)
    elif op == "layernorm":
        st = rw.rowop_layernorm_backward(x.data_ptr(), x.data_ptr(), None, x.data_ptr(), None,
                                         None, 1, cap + 1, cap + 1, F32, 1e-5, None, 0, s)
    else:
        st = rw.rowop_rmsnorm_backward(x.data_ptr(), x.data_ptr(), None, x.data_ptr(), None,
                                       1, cap + 1, cap + 1, F32, 1e-6, None, 0, s)
    assert st == rw.ROWOP_ERR_TOO_LONG


@pytest.mark.parametrize("dtype", DTYPES, ids=DTYPE_IDS)
@pytest.mark.parametrize("op", OPS)
@pytest.mark.parametrize("cols,ld,offs", [
    (777, 777, (1, 1, 1)),      # congruent, every row starts mid-chunk: vector path with edges
    (5000, 5008, (3, 3, 3)),
    (777, 777, (0, 1, 0)),      # dy not congruent: element path
    (3001, 3003, (0, 0, 0)),    # ld not a whole number of chunks: element path
    (20000, 20001, (2, 5, 1)),  # element path over a cluster
])
def test_backward_misaligned(rw, op, dtype, cols, ld, offs):
    run_bwd(rw, op, dtype, 6, cols, ld=ld, offs=offs, seed=cols + ld)


@pytest.mark.parametrize("op", OPS)
@pytest.mark.parametrize("where", ["dy", "a"])
@pytest.mark.parametrize("cols", [300, 4096, 30000])
def test_backward_inplace(rw, op, where, cols):
    run_bwd(rw, op, torch.bfloat16, 7, cols, inplace=where, seed=4)


@pytest.mark.parametrize("op", NORMS)
def test_backward_param_options(rw, op):
    """dgamma / dbeta each optional, gamma optional."""
    for want in ((True, False), (False, True), (False, False)):
        run_bwd(rw, op, torch.float32, 40, 1500, want=want, seed=11)
    run_bwd(rw, op, torch.float32, 40, 1500, affine=False, seed=12)


@pytest.mark.parametrize("op", NORMS)
def test_backward_zero_rows_zero_params(rw, op):
    """No rows: dgamma / dbeta are sums over nothing, written as zeros."""
    _, dg, db = run_bwd(rw, op, torch.float32, 0, 300, compare=False)
    assert (dg.cpu() == 0).all()
    if op == "layernorm":
        assert (db.cpu() == 0).all()


@pytest.mark.parametrize("dtype", DTYPES, ids=DTYPE_IDS)
@pytest.mark.parametrize("op", OPS)
@pytest.mark.parametrize("rows,cols", [(20000, 64), (3000, 300), (2500, 1024)])
def test_backward_many_rows(rw, op, dtype, rows, cols):
    """Many rows per team and many teams per CTA: the dgamma / dbeta partials
    and their sums."""
    run_bwd(rw, op, dtype, rows, cols, seed=rows)


@pytest.mark.parametrize("op", OPS)
@pytest.mark.parametrize("cs", [2, 4, 16])
def test_backward_forced_cluster(rw, op, cs, monkeypatch):
    """The cluster exchange on rows that one CTA could hold."""
    monkeypatch.setenv("ROWOP_BWD_CLUSTER", str(cs))
    for cols, rows in ((3000, 9), (9000, 40)):
        run_bwd(rw, op, torch.float32, rows, cols, seed=cols + cs)
        run_bwd(rw, op, torch.bfloat16, rows, cols, offs=(1, 1, 1), seed=cols + cs)


@pytest.mark.parametrize("cols", [100, 4096, 40000])
@pytest.mark.parametrize("mean,std", [(100.0, 1.0), (-5.0, 0.05)])
def test_layernorm_backward_far_from_zero(rw, cols, mean, std):
    """fp32 LayerNorm backward of rows whose mean is 100 times their spread
    (several teams per CTA, one team per CTA, cluster-split rows): the row
    statistics, merged pairwise from each thread's own, keep the full
    tolerance (a one-pass E[x^2] - mean^2 would lose about 100^2 * 2^-24 of
    the variance).  Far larger ratios are bounded by the fp32 mean itself,
    whose rounding shifts every xhat by up to ulp(mean) / (2 std)."""
    dtype = torch.float32
    g = torch.Generator("cpu").manual_seed(cols)
    x = (mean + std * torch.randn(6, cols, generator=g, dtype=torch.float64)).float()
    dy = torch.randn(6, cols, generator=g)
    gam = 1.0 + 0.2 * torch.randn(cols, generator=g)
    dx, dg, db = rw.layernorm_backward(x.cuda(), dy.cuda(), gam.cuda(), 1e-5)
    assert rw.check_status() == 0
    a64, d64, g64 = x.double().numpy(), dy.double().numpy(), gam.double().numpy()
    eps = float(np.float32(1e-5))
    rdx, rdg, rdb = oracle("layernorm", a64, d64, g64, eps)
    sdx, sdg, sdb = scales("layernorm", a64, d64, g64, eps)
    what = f"layernorm far from zero (mean {mean}, std {std}, {cols} cols)"
    check(to_f64(dx), rdx, sdx, dtype, R_COMP, what + " dx")
    check(to_f64(dg), rdg, sdg, dtype, R_COMP_PARAM, what + " dgamma")
    check(to_f64(db), rdb, sdb, dtype, R_COMP_PARAM, what + " dbeta")


@pytest.mark.parametrize("op", OPS)
def test_backward_deterministic(rw, op):
    outs = [run_bwd(rw, op, torch.bfloat16, 700, 5000, seed=5, compare=(i == 0)) for i in range(2)]
    assert torch.equal(_bits(outs[0][0]), _bits(outs[1][0]))
    for k in (1, 2):
        if outs[0][k] is not None:
            assert torch.equal(_bits(outs[0][k]), _bits(outs[1][k]))


def test_backward_binding(rw):
    """The torch helpers allocate outputs and workspace and agree with the C
    calls."""
    a, dy, gam = inputs("layernorm", torch.bfloat16, 64, 2048, 3)
    dx, dg, db = rw.layernorm_backward(a.cuda(), dy.cuda(), gam.cuda(), 1e-5)
    ref_dx, ref_dg, ref_db = orc.layernorm_backward(a.double().numpy(), dy.double().numpy(),
                                                    gam.double().numpy(),
                                                    eps=float(np.float32(1e-5)))
    s_dx, s_dg, s_db = scales("layernorm", a.double().numpy(), dy.double().numpy(),
                              gam.double().numpy(), float(np.float32(1e-5)))
    check(to_f64(dx), ref_dx, s_dx, torch.bfloat16, R_COMP, "binding dx")
    check(to_f64(dg), ref_dg, s_dg, torch.bfloat16, R_COMP_PARAM, "binding dgamma")
    check(to_f64(db), ref_db, s_db, torch.bfloat16, R_COMP_PARAM, "binding dbeta")
    y = torch.from_numpy(orc.softmax(np.random.default_rng(0).normal(size=(8, 100)))).float()
    d = torch.randn(8, 100)
    got = rw.softmax_backward(y.cuda(), d.cuda())
    check(to_f64(got), orc.softmax_backward(y.double().numpy(), d.double().numpy()),
          scales("softmax", y.double().numpy(), d.double().numpy(), None, 0)[0],
          torch.float32, R_COMP, "binding softmax dx")


@pytest.mark.parametrize("op", NORMS)
def test_workload_norm_backward(rw, op):
    """The bf16 norm-backward workload at full size (8192 x 4096), called as
    the benchmark calls it: dx on every 32nd row, dgamma / dbeta over all
    rows."""
    from paper_2607_23089_gb300 import workloads as wl
    case = wl.norm_backward(op)
    x, dy, gam = case.x.cuda(), case.dy.cuda(), case.gamma.cuda()
    if op == "layernorm":
        dx, dg, db = rw.layernorm_backward(x, dy, gam, case.eps)
    else:
        (dx, dg), db = rw.rmsnorm_backward(x, dy, gam, case.eps), None
    assert rw.check_status() == 0
    a64, dy64, g64 = case.x.double().numpy(), case.dy.double().numpy(), case.gamma.double().numpy()
    eps = float(np.float32(case.eps))
    ref_dx, ref_dg, ref_db = oracle(op, a64, dy64, g64, eps)
    s_dx, s_dg, s_db = scales(op, a64, dy64, g64, eps)
    sel = slice(None, None, 32)
    check(to_f64(dx[sel]), ref_dx[sel], s_dx[sel], case.dtype, R_COMP, f"{case.name} dx")
    check(to_f64(dg), ref_dg, s_dg, case.dtype, R_COMP_PARAM, f"{case.name} dgamma")
    if op == "layernorm":
        check(to_f64(db), ref_db, s_db, case.dtype, R_COMP_PARAM, f"{case.name} dbeta")


@pytest.mark.parametrize("op", ["softmax", "logsoftmax"])
def test_workload_softmax_backward(rw, op):
    """The fp32 softmax-family backward workload at full size (32768 x 1024);
    y is the oracle's forward of the workload's x, rounded to fp32; dx
    checked on every 16th row."""
    from paper_2607_23089_gb300 import workloads as wl
    case = wl.softmax_backward(op)
    x64 = case.x.double().numpy()
    y = torch.from_numpy(orc.softmax(x64, nthreads=8) if op == "softmax"
                         else orc.logsoftmax(x64, nthreads=8)).float()
    dx = rw.run(f"{op}_backward", y.cuda(), dy=case.dy.cuda())
    assert rw.check_status() == 0
    sel = slice(None, None, 16)
    a64, dy64 = y[sel].double().numpy(), case.dy[sel].double().numpy()
    ref = (orc.softmax_backward if op == "softmax" else orc.logsoftmax_backward)(a64, dy64)
    check(to_f64(dx[sel]), ref, scales(op, a64, dy64, None, 0)[0], case.dtype, R_COMP,
          f"{case.name} dx")


def _ragged_lengths(dtype, rows, seed, max_len):
    """Lengths over all three row buckets, with empty and length-1 rows."""
    es = ESIZE[dtype]
    g = np.random.default_rng(seed)
    pools = [(0, 1), (1, 40), (41, 4096 // es), (4096 // es + 1, 32768 // es),
             (32768 // es + 1, max_len)]
    lens = [int(g.integers(lo, max(lo, min(hi, max_len)) + 1)) for lo, hi in
            (pools[i % len(pools)] for i in range(rows))]
    g.shuffle(lens)
    return np.array(lens, dtype=np.int64)


def run_bwd_ragged(rw, op, dtype, lens, max_len, seed, base_off=0, inplace=False):
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64) + base_off
    total = int(off[-1])
    rows = len(lens)
    g = torch.Generator("cpu").manual_seed(seed)
    y = torch.zeros(total, dtype=torch.float64)
    for i in range(rows):
        if lens[i]:
            x = (3.0 * torch.randn(1, int(lens[i]), generator=g, dtype=torch.float64)).numpy()
            y[off[i]:off[i + 1]] = torch.from_numpy(
                (orc.softmax(x) if op == "softmax" else orc.logsoftmax(x))[0])
    y = y.to(dtype)
    dy = torch.randn(total, generator=g).to(dtype)
    yb = canary_tensor(G + total + G, dtype)
    yb[G:G + total] = y.cuda()
    db = canary_tensor(G + total + G, dtype)
    db[G:G + total] = dy.cuda()
    xb = db if inplace else canary_tensor(G + total + G, dtype)
    es = ESIZE[dtype]
    offd = torch.from_numpy(off).cuda()
    ws = rw.ragged_workspace(rows)
    fn = rw.rowop_softmax_backward_ragged if op == "softmax" else rw.rowop_logsoftmax_backward_ragged
    st = fn(yb.data_ptr() + G * es, db.data_ptr() + G * es, xb.data_ptr() + G * es,
            offd.data_ptr(), rows, max_len, rw.dtype_code(dtype), ws.data_ptr(), ws.numel(),
            torch.cuda.current_stream().cuda_stream)
    assert st == 0, rw.STATUS.get(st, st)
    return y, dy, xb, off, st


@pytest.mark.parametrize("dtype", DTYPES, ids=DTYPE_IDS)
@pytest.mark.parametrize("op", ["softmax", "logsoftmax"])
@pytest.mark.parametrize("base_off", [0, 3])
def test_backward_ragged(rw, op, dtype, base_off):
    """Ragged softmax-family backward against the oracle row by row; rows of
    every bucket (cluster-split ones included), empty and one-element rows,
    rows at every alignment; nothing outside the rows is written."""
    max_len = 70000
    lens = _ragged_lengths(dtype, 60, 5, max_len)
    y, dy, xb, off, _ = run_bwd_ragged(rw, op, dtype, lens, max_len, seed=9, base_off=base_off)
    assert rw.check_status() == 0
    dx = to_f64(xb[G:G + int(off[-1])])
    for i, n in enumerate(lens):
        if n == 0:
            continue
        a64 = y[off[i]:off[i + 1]].double().numpy()[None, :]
        d64 = dy[off[i]:off[i + 1]].double().numpy()[None, :]
        ref = (orc.softmax_backward if op == "softmax" else orc.logsoftmax_backward)(a64, d64)
        check(dx[None, off[i]:off[i + 1]], ref, scales(op, a64, d64, None, 0)[0], dtype, R_COMP,
              f"ragged {op} row {i} (len {n})")
    assert is_canary(xb[:G + base_off]).all() and is_canary(xb[G + int(off[-1]):]).all()


@pytest.mark.parametrize("op", ["softmax", "logsoftmax"])
def test_backward_ragged_inplace_and_rejects(rw, op):
    """dx written over dy; a row longer than max_len is skipped, left as it
    was and flagged, while the other rows are still done."""
    dtype = torch.float32
    lens = np.array([5, 300, 2000, 9000, 40], dtype=np.int64)
    y, dy, xb, off, _ = run_bwd_ragged(rw, op, dtype, lens, 8000, seed=2, inplace=True)
    assert rw.check_status() == rw.ROWOP_ERR_BAD_OFFSETS
    got = to_f64(xb[G:G + int(off[-1])])
    # the 9000-element row is longer than max_len: its dy is untouched
    assert np.array_equal(got[off[3]:off[4]], dy[off[3]:off[4]].double().numpy())
    for i in (0, 1, 2, 4):
        a64 = y[off[i]:off[i + 1]].double().numpy()[None, :]
        d64 = dy[off[i]:off[i + 1]].double().numpy()[None, :]
        ref = (orc.softmax_backward if op == "softmax" else orc.logsoftmax_backward)(a64, d64)
        check(got[None, off[i]:off[i + 1]], ref, scales(op, a64, d64, None, 0)[0], dtype, R_COMP,
              f"ragged {op} row {i}")


def test_workload_ragged_softmax_backward(rw):
    """The ragged softmax-backward workload at full size (32768 rows, lengths
    up to 4096), y the oracle's forward of the workload's x rounded to fp32;
    dx checked on every 64th row."""
    from paper_2607_23089_gb300 import workloads as wl
    case = wl.ragged_softmax_backward()
    off = case.offsets.numpy()
    y = torch.from_numpy(orc.softmax_ragged(case.x.double().numpy(), off, nthreads=8)).float()
    offd = case.offsets.cuda()
    dx = rw.softmax_backward_ragged(y.cuda(), case.dy.cuda(), offd, case.max_len)
    assert rw.check_status() == 0
    got = to_f64(dx)
    for i in range(0, case.rows, 64):
        a64 = y[off[i]:off[i + 1]].double().numpy()[None, :]
        d64 = case.dy[off[i]:off[i + 1]].double().numpy()[None, :]
        check(got[None, off[i]:off[i + 1]], orc.softmax_backward(a64, d64),
              scales("softmax", a64, d64, None, 0)[0], torch.float32, R_COMP,
              f"ragged softmax backward workload row {i}")


# rows of whole 1 KiB tiles that the whole-tile norm kernel takes: 4, 8 and
# 16 warps of one tile (16-bit types) or two tiles (fp32) each
WHOLE_TILE_COLS = {4: (2048, 4096, 8192), 2: (2048, 4096, 8192)}


@pytest.mark.parametrize("dtype", DTYPES, ids=DTYPE_IDS)
@pytest.mark.parametrize("op", NORMS)
def test_backward_whole_tile_rows(rw, op, dtype, monkeypatch):
    """The whole-tile design (x and dy staged by bulk copies, gamma and the
    dgamma / dbeta sums in registers) and the team design both hold the
    oracle's tolerance: few rows (fewer than the stages), many rows per CTA
    (the stage ring wraps many times), a row stride wider than the row, and
    no gamma."""
    es = ESIZE[dtype]
    for cols in WHOLE_TILE_COLS[es]:
        for tile in ("1", "0"):
            monkeypatch.setenv("ROWOP_BWD_TILE", tile)
            run_bwd(rw, op, dtype, 3, cols, seed=cols + 1)
            run_bwd(rw, op, dtype, 1500 if cols < 8192 else 700, cols, seed=cols + 2)
            run_bwd(rw, op, dtype, 37, cols, ld=cols + 64, seed=cols + 3)
            run_bwd(rw, op, dtype, 37, cols, affine=False, seed=cols + 4)


@pytest.mark.parametrize("op", NORMS)
def test_backward_whole_tile_options(rw, op):
    """dgamma / dbeta each optional, in place over x or dy, and rows that are
    not 16-byte aligned (the team design takes those) on the same shape."""
    for want in ((True, False), (False, True), (False, False)):
        run_bwd(rw, op, torch.bfloat16, 300, 4096, want=want, seed=21)
    for where in ("dy", "a"):
        run_bwd(rw, op, torch.bfloat16, 300, 4096, inplace=where, seed=22)
    run_bwd(rw, op, torch.bfloat16, 30, 4096, offs=(8, 8, 8), seed=23)
    run_bwd(rw, op, torch.bfloat16, 30, 4096, offs=(1, 1, 1), seed=24)


@pytest.mark.parametrize("op", NORMS)
def test_backward_whole_tile_deterministic(rw, op):
    outs = [run_bwd(rw, op, torch.bfloat16, 2000, 4096, seed=5, compare=(i == 0))
            for i in range(2)]
    for k in (0, 1, 2):
        if outs[0][k] is not None:
            assert torch.equal(_bits(outs[0][k]), _bits(outs[1][k]))
