"""GPU parity of the ragged LayerNorm / RMSNorm backward passes through the C
ABI, against the double-precision oracle (the dense backward of each row,
dgamma / dbeta summed over the rows that reach each column), with the
tolerance the dense backward tests derive: r_out * |ref| + r_comp * S + a_out,
r_comp = 1e-5 for dx and 3e-5 for dgamma / dbeta."""
import numpy as np
import pytest
import torch

from oracle import rowop_oracle as orc
from tests.gpu_util import DTYPE_IDS, DTYPES, ESIZE, canary_tensor, is_canary, to_f64
from tests.test_gpu_backward import R_COMP, R_COMP_PARAM, _ragged_lengths, check, scales

pytestmark = pytest.mark.gpu
G = 64
EPS = {"layernorm": 1e-5, "rmsnorm": 1e-6}


@pytest.fixture(scope="module")
def rw():
    from paper_2607_23089_gb300 import build, rowop
    build.build()
    rowop.load()
    torch.cuda.set_device(0)
    return rowop


def make_inputs(dtype, lens, max_len, seed, base_off=0, affine=True):
    """x (a scale and shift per row), dy = N(0,1) and gamma of max_len, packed
    after base_off unused elements."""
    off = (np.concatenate([[0], np.cumsum(lens)]) + base_off).astype(np.int64)
    total = int(off[-1])
    g = torch.Generator("cpu").manual_seed(seed)
    rows = len(lens)
    scale = 0.2 + 5.0 * torch.rand(rows, generator=g, dtype=torch.float64)
    shift = 2.0 * torch.randn(rows, generator=g, dtype=torch.float64)
    per = torch.repeat_interleave(torch.arange(rows), torch.from_numpy(np.asarray(lens)))
    x = torch.zeros(total, dtype=torch.float64)
    x[base_off:] = torch.randn(total - base_off, generator=g, dtype=torch.float64) * scale[per] + shift[per]
    dy = torch.randn(total, generator=g)
    gam = (1.0 + 0.2 * torch.randn(max(max_len, 1), generator=g)) if affine else None
    return x.to(dtype), dy.to(dtype), None if gam is None else gam.to(dtype), off


def call(rw, op, dtype, x, dy, gam, off, max_len, inplace=None, want=(True, True), shift=0):
    """One call on canary-guarded buffers; returns (status, dx buffer, dgamma
    buffer, dbeta buffer) -- the data sits at [G, G + n) of each.  x, dy and
    dx start `shift` elements past G of their allocations (the returned dx
    buffer is the view from `shift`)."""
    total = int(off[-1])
    rows = len(off) - 1
    es = ESIZE[dtype]
    xb = canary_tensor(shift + G + total + G, dtype)[shift:]
    xb[G:G + total] = x.cuda()
    db = canary_tensor(shift + G + total + G, dtype)[shift:]
    db[G:G + total] = dy.cuda()
    if inplace == "dy":
        dxb = db
    elif inplace == "x":
        dxb = xb
    else:
        dxb = canary_tensor(shift + G + total + G, dtype)[shift:]
    n = max(max_len, 1)
    dgb = canary_tensor(G + n + G, dtype) if want[0] else None
    dbb = canary_tensor(G + n + G, dtype) if (op == "layernorm" and want[1]) else None
    gd = gam.cuda() if gam is not None else None
    offd = torch.from_numpy(off).cuda()
    code = rw.dtype_code(dtype)
    size_fn = (rw.rowop_layernorm_backward_ragged_workspace_size if op == "layernorm"
               else rw.rowop_rmsnorm_backward_ragged_workspace_size)
    ws = torch.empty(int(size_fn(rows, max_len, code)), dtype=torch.uint8, device="cuda")
    p = lambda b: None if b is None else b.data_ptr() + G * es  # noqa: E731
    s = torch.cuda.current_stream().cuda_stream
    gp = None if gd is None else gd.data_ptr()
    if op == "layernorm":
        st = rw.rowop_layernorm_backward_ragged(p(xb), p(db), gp, p(dxb), p(dgb), p(dbb),
                                                offd.data_ptr(), rows, max_len, code, EPS[op],
                                                ws.data_ptr(), ws.numel(), s)
    else:
        st = rw.rowop_rmsnorm_backward_ragged(p(xb), p(db), gp, p(dxb), p(dgb), offd.data_ptr(),
                                              rows, max_len, code, EPS[op], ws.data_ptr(),
                                              ws.numel(), s)
    torch.cuda.synchronize()
    return st, dxb, dgb, dbb


def reference(op, x, dy, gam, off, max_len, skip=()):
    """Oracle dx rows and dgamma / dbeta over max_len columns, with their
    tolerance scales; rows in `skip` left out."""
    eps = float(np.float32(EPS[op]))
    rows = len(off) - 1
    x64, d64 = x.double().numpy(), dy.double().numpy()
    g64 = np.ones(max(max_len, 1)) if gam is None else gam.double().numpy()
    keep = [i for i in range(rows) if i not in skip]
    sub_off = np.concatenate([[0], np.cumsum([off[i + 1] - off[i] for i in keep])]).astype(np.int64)
    xs = np.concatenate([x64[off[i]:off[i + 1]] for i in keep] + [np.zeros(0)])
    ds = np.concatenate([d64[off[i]:off[i + 1]] for i in keep] + [np.zeros(0)])
    fn = orc.layernorm_backward_ragged if op == "layernorm" else orc.rmsnorm_backward_ragged
    out = fn(xs, ds, sub_off, g64, eps=eps)
    dx_rows, sdg, sdb = {}, np.zeros(max_len), np.zeros(max_len)
    for k, i in enumerate(keep):
        a, b = int(sub_off[k]), int(sub_off[k + 1])
        if b == a:
            continue
        s_dx, s_g, s_b = scales(op, xs[None, a:b], ds[None, a:b], g64[:b - a], eps)
        dx_rows[i] = (out[0][a:b], s_dx[0])
        sdg[:b - a] += s_g
        sdb[:b - a] += s_b
    pads = [np.pad(v, (0, max_len - v.shape[0])) for v in out[1:]]
    return dx_rows, pads, (sdg, sdb)


def verify(op, dtype, dx_rows, params, pscales, off, dxb, dgb, dbb, max_len, what):
    total = int(off[-1])
    got = to_f64(dxb[G:G + total])
    for i, (ref, s) in dx_rows.items():
        check(got[None, off[i]:off[i + 1]], ref[None], s[None], dtype, R_COMP, f"{what} dx row {i}")
    for buf, ref, s, name in ((dgb, params[0], pscales[0], "dgamma"),
                              (dbb, params[1] if len(params) > 1 else None, pscales[1], "dbeta")):
        if buf is None:
            continue
        check(to_f64(buf[G:G + max_len]), ref, s, dtype, R_COMP_PARAM, f"{what} {name}")
        assert is_canary(buf[:G]).all() and is_canary(buf[G + max_len:]).all(), f"{what} {name}"


@pytest.mark.parametrize("dtype", DTYPES, ids=DTYPE_IDS)
@pytest.mark.parametrize("op", ["layernorm", "rmsnorm"])
@pytest.mark.parametrize("base_off", [0, 5])
@pytest.mark.parametrize("design", ["team", "stripe"])
def test_ragged_norm_backward(rw, monkeypatch, op, dtype, base_off, design):
    """Rows of every bucket (cluster-split ones included), empty and
    one-element rows, every alignment; dgamma / dbeta over max_len columns,
    the last ones past every row (zero); nothing outside the outputs
    written.  Both designs: the bucket launches of the team kernel and the
    column stripes."""
    monkeypatch.setenv("ROWOP_BWD_STRIPE", "0" if design == "team" else "1")
    lens = _ragged_lengths(dtype, 60, 6, 70000)
    max_len = int(lens.max()) + 37
    x, dy, gam, off = make_inputs(dtype, lens, max_len, seed=11, base_off=base_off)
    st, dxb, dgb, dbb = call(rw, op, dtype, x, dy, gam, off, max_len)
    assert st == 0, rw.STATUS.get(st, st)
    assert rw.check_status() == 0
    dx_rows, params, ps = reference(op, x, dy, gam, off, max_len)
    verify(op, dtype, dx_rows, params, ps, off, dxb, dgb, dbb, max_len, f"{op} {dtype}")
    assert (to_f64(dgb[G + int(lens.max()):G + max_len]) == 0).all()
    assert is_canary(dxb[:G + base_off]).all() and is_canary(dxb[G + int(off[-1]):]).all()


@pytest.mark.parametrize("op", ["layernorm", "rmsnorm"])
@pytest.mark.parametrize("max_len", [1, 40, 2048, 2049, 16384, 16385, 100000, 131072])
def test_ragged_norm_backward_bucket_edges(rw, op, max_len):
    """max_len at and around the bucket edges of bf16 (launch covers of one,
    two or three buckets) and at the longest ragged norm row, rows up to
    max_len."""
    dtype = torch.bfloat16
    g = np.random.default_rng(max_len)
    lens = np.minimum(max_len, g.integers(0, max_len + 1, 24)).astype(np.int64)
    lens[0] = max_len
    x, dy, gam, off = make_inputs(dtype, lens, max_len, seed=max_len)
    st, dxb, dgb, dbb = call(rw, op, dtype, x, dy, gam, off, max_len)
    assert st == 0 and rw.check_status() == 0
    dx_rows, params, ps = reference(op, x, dy, gam, off, max_len)
    verify(op, dtype, dx_rows, params, ps, off, dxb, dgb, dbb, max_len, f"{op} max_len {max_len}")


@pytest.mark.parametrize("op", ["layernorm", "rmsnorm"])
def test_ragged_norm_backward_options(rw, op):
    """gamma NULL (ones); only dgamma; no parameter gradients; dx over dy and
    over x."""
    dtype = torch.float32
    lens = _ragged_lengths(dtype, 30, 8, 20000)
    max_len = int(lens.max())
    x, dy, gam, off = make_inputs(dtype, lens, max_len, seed=12, affine=False)
    dx_rows, params, ps = reference(op, x, dy, None, off, max_len)
    for inplace, want in ((None, (True, True)), (None, (True, False)), ("dy", (False, False)),
                          ("x", (True, True))):
        st, dxb, dgb, dbb = call(rw, op, dtype, x, dy, None, off, max_len, inplace, want)
        assert st == 0 and rw.check_status() == 0
        verify(op, dtype, dx_rows, params, ps, off, dxb, dgb, dbb, max_len,
               f"{op} inplace {inplace} want {want}")


@pytest.mark.parametrize("op", ["layernorm", "rmsnorm"])
def test_ragged_norm_backward_zero_rows(rw, op):
    """No rows: dgamma / dbeta of max_len columns are set to zero."""
    dtype = torch.bfloat16
    max_len = 3000
    dg = torch.full((max_len,), 7.0, dtype=dtype, device="cuda")
    db = torch.full((max_len,), 7.0, dtype=dtype, device="cuda")
    off = torch.zeros(1, dtype=torch.int64, device="cuda")
    code = rw.dtype_code(dtype)
    s = torch.cuda.current_stream().cuda_stream
    if op == "layernorm":
        size = rw.rowop_layernorm_backward_ragged_workspace_size(0, max_len, code)
        ws = torch.empty(int(size), dtype=torch.uint8, device="cuda")
        st = rw.rowop_layernorm_backward_ragged(None, None, None, None, dg.data_ptr(),
                                                db.data_ptr(), off.data_ptr(), 0, max_len, code,
                                                1e-5, ws.data_ptr(), ws.numel(), s)
    else:
        size = rw.rowop_rmsnorm_backward_ragged_workspace_size(0, max_len, code)
        ws = torch.empty(int(size), dtype=torch.uint8, device="cuda")
        st = rw.rowop_rmsnorm_backward_ragged(None, None, None, None, dg.data_ptr(),
                                              off.data_ptr(), 0, max_len, code, 1e-6,
                                              ws.data_ptr(), ws.numel(), s)
    assert st == 0
    torch.cuda.synchronize()
    assert (dg == 0).all()
    if op == "layernorm":
        assert (db == 0).all()


@pytest.mark.parametrize("op", ["layernorm", "rmsnorm"])
def test_ragged_norm_backward_rejects(rw, op):
    """A row longer than max_len is skipped (dx left as it was) and flagged;
    the other rows are done, and dgamma / dbeta leave the skipped row out."""
    dtype = torch.float32
    lens = np.array([5, 300, 2000, 9000, 40, 0, 7000], dtype=np.int64)
    max_len = 8000
    x, dy, gam, off = make_inputs(dtype, lens, max_len, seed=13)
    st, dxb, dgb, dbb = call(rw, op, dtype, x, dy, gam, off, max_len, inplace="dy")
    assert st == 0
    assert rw.check_status() == rw.ROWOP_ERR_BAD_OFFSETS
    got = to_f64(dxb[G:G + int(off[-1])])
    assert np.array_equal(got[off[3]:off[4]], dy[off[3]:off[4]].double().numpy())
    dx_rows, params, ps = reference(op, x, dy, gam, off, max_len, skip=(3,))
    verify(op, dtype, dx_rows, params, ps, off, dxb, dgb, dbb, max_len, f"{op} rejects")


@pytest.mark.parametrize("op", ["layernorm", "rmsnorm"])
def test_ragged_norm_backward_deterministic(rw, op):
    """Two calls on the same input give the same bits."""
    dtype = torch.bfloat16
    lens = _ragged_lengths(dtype, 80, 14, 40000)
    max_len = int(lens.max())
    x, dy, gam, off = make_inputs(dtype, lens, max_len, seed=14)
    a = call(rw, op, dtype, x, dy, gam, off, max_len)
    b = call(rw, op, dtype, x, dy, gam, off, max_len)
    for u, v in zip(a[1:], b[1:]):
        if u is not None:
            assert torch.equal(u.view(torch.int16), v.view(torch.int16))


def test_ragged_norm_backward_binding(rw):
    """The Python helpers allocate what is not given and return the
    gradients."""
    dtype = torch.bfloat16
    lens = np.array([3, 0, 700, 5000], dtype=np.int64)
    max_len = 5000
    x, dy, gam, off = make_inputs(dtype, lens, max_len, seed=15)
    offd = torch.from_numpy(off).cuda()
    dx, dg, db = rw.layernorm_backward_ragged(x.cuda(), dy.cuda(), offd, max_len, gam.cuda())
    assert rw.check_status() == 0
    dx_rows, params, ps = reference("layernorm", x, dy, gam, off, max_len)
    got = to_f64(dx)
    for i, (ref, s) in dx_rows.items():
        check(got[None, off[i]:off[i + 1]], ref[None], s[None], dtype, R_COMP, f"binding dx row {i}")
    check(to_f64(dg), params[0], ps[0], dtype, R_COMP_PARAM, "binding dgamma")
    check(to_f64(db), params[1], ps[1], dtype, R_COMP_PARAM, "binding dbeta")
    dx, dg = rw.rmsnorm_backward_ragged(x.cuda(), dy.cuda(), offd, max_len, gam.cuda(),
                                        want_dgamma=False)
    assert dg is None


@pytest.mark.parametrize("op", ["layernorm", "rmsnorm"])
def test_workload_ragged_norm_backward(rw, op):
    """The ragged norm-backward workload at full size (16384 bf16 rows,
    lengths uniform on 1..32768, one launch per bucket as the benchmark times
    it): dx on every 64th row, dgamma / dbeta on every column against the
    oracle over all rows (taken in row chunks)."""
    from paper_2607_23089_gb300 import workloads as wl
    case = wl.ragged_norm_backward(op)
    off = case.offsets.numpy()
    xd, dyd, gd = case.x.cuda(), case.dy.cuda(), case.gamma.cuda()
    offd = case.offsets.cuda()
    fn = rw.layernorm_backward_ragged if op == "layernorm" else rw.rmsnorm_backward_ragged
    out = fn(xd, dyd, offd, case.max_len, gd, case.eps)
    assert rw.check_status() == 0
    dx = to_f64(out[0])
    eps = float(np.float32(case.eps))
    g64 = case.gamma.double().numpy()
    sums = [np.zeros(case.max_len) for _ in out[1:]]
    ssum = [np.zeros(case.max_len) for _ in out[1:]]
    ofn = orc.layernorm_backward_ragged if op == "layernorm" else orc.rmsnorm_backward_ragged
    step = 1024
    for r0 in range(0, case.rows, step):
        r1 = min(case.rows, r0 + step)
        a, b = int(off[r0]), int(off[r1])
        xs = case.x[a:b].double().numpy()
        ds = case.dy[a:b].double().numpy()
        res = ofn(xs, ds, off[r0:r1 + 1] - a, g64, eps=eps)
        for s, part in zip(sums, res[1:]):
            s[:part.shape[0]] += part
        for i in range(r0, r1):
            lo, hi = int(off[i]) - a, int(off[i + 1]) - a
            sc = scales(op, xs[None, lo:hi], ds[None, lo:hi], g64[:hi - lo], eps)
            for s, part in zip(ssum, sc[1:]):
                s[:hi - lo] += part
            if i % 64 == 0:
                check(dx[None, off[i]:off[i + 1]], res[0][None, lo:hi], sc[0], case.dtype, R_COMP,
                      f"workload {op} dx row {i}")
    for k, name in enumerate(("dgamma", "dbeta")[:len(sums)]):
        check(to_f64(out[1 + k]), sums[k], ssum[k], case.dtype, R_COMP_PARAM, f"workload {name}")


def _stripe_widths(dtype):
    """Window positions of a stripe of the stats and dx kernels: 512 and 256
    chunks of 16 bytes (a stripe's columns move with the row's head
    offset)."""
    e = 16 // ESIZE[dtype]
    return e * 512, e * 256


@pytest.mark.parametrize("dtype", DTYPES, ids=DTYPE_IDS)
@pytest.mark.parametrize("op", ["layernorm", "rmsnorm"])
@pytest.mark.parametrize("base_off", [0, 3])
def test_ragged_norm_backward_stripe_edges(rw, monkeypatch, op, dtype, base_off):
    """The column-stripe design, taken for every max_len: rows that end at,
    one before and one past the stripe edges of both kernels, rows shorter
    than a chunk, empty and one-element rows, at every head class (the
    lengths repeat, so each length lands at several starts); against the
    oracle, with nothing outside the outputs written."""
    monkeypatch.setenv("ROWOP_BWD_STRIPE", "2")
    w1, w2 = _stripe_widths(dtype)
    base = [0, 1, 2, 3, 5, 7, 8, 9, 15, 17, w2 - 7, w2 - 1, w2, w2 + 1, w2 + 7, 2 * w2 + 3,
            w1 - 7, w1 - 1, w1, w1 + 1, w1 + 7, w1 + w2, 2 * w1 + 5]
    lens = np.array(base * 3, dtype=np.int64)
    np.random.default_rng(base_off).shuffle(lens)
    max_len = int(lens.max()) + 11
    x, dy, gam, off = make_inputs(dtype, lens, max_len, seed=21, base_off=base_off)
    st, dxb, dgb, dbb = call(rw, op, dtype, x, dy, gam, off, max_len)
    assert st == 0 and rw.check_status() == 0
    dx_rows, params, ps = reference(op, x, dy, gam, off, max_len)
    verify(op, dtype, dx_rows, params, ps, off, dxb, dgb, dbb, max_len, f"stripe {op} {dtype}")
    assert is_canary(dxb[:G + base_off]).all() and is_canary(dxb[G + int(off[-1]):]).all()


@pytest.mark.parametrize("op", ["layernorm", "rmsnorm"])
@pytest.mark.parametrize("max_len", [1, 9, 300])
def test_ragged_norm_backward_stripe_short(rw, monkeypatch, op, max_len):
    """The column-stripe design on short rows (one stripe, mostly idle lanes),
    the options of the call (gamma NULL, dgamma only, no parameter
    gradients, dx over dy and over x) and a rejected row."""
    monkeypatch.setenv("ROWOP_BWD_STRIPE", "2")
    dtype = torch.float32
    g = np.random.default_rng(max_len)
    lens = g.integers(0, max_len + 1, 70).astype(np.int64)
    x, dy, gam, off = make_inputs(dtype, lens, max_len, seed=22, affine=False)
    dx_rows, params, ps = reference(op, x, dy, None, off, max_len)
    for inplace, want in ((None, (True, True)), (None, (True, False)), ("dy", (False, False)),
                          ("x", (True, True))):
        st, dxb, dgb, dbb = call(rw, op, dtype, x, dy, None, off, max_len, inplace, want)
        assert st == 0 and rw.check_status() == 0
        verify(op, dtype, dx_rows, params, ps, off, dxb, dgb, dbb, max_len,
               f"stripe short {op} max_len {max_len} inplace {inplace} want {want}")
    lens2 = lens.copy()
    lens2[3] = max_len + 1
    x, dy, gam, off = make_inputs(dtype, lens2, max_len, seed=23)
    st, dxb, dgb, dbb = call(rw, op, dtype, x, dy, gam, off, max_len, inplace="dy")
    assert st == 0
    assert rw.check_status() == rw.ROWOP_ERR_BAD_OFFSETS
    got = to_f64(dxb[G:G + int(off[-1])])
    assert np.array_equal(got[off[3]:off[4]], dy[off[3]:off[4]].double().numpy())
    dx_rows, params, ps = reference(op, x, dy, gam, off, max_len, skip=(3,))
    verify(op, dtype, dx_rows, params, ps, off, dxb, dgb, dbb, max_len, f"stripe rejects {op}")


def test_ragged_norm_backward_stripe_many_rows(rw, monkeypatch):
    """More rows than the dx kernel's groups take in one sorted batch (33000
    rows: 128 groups of 258), in both designs, against the oracle."""
    dtype = torch.bfloat16
    g = np.random.default_rng(24)
    lens = g.integers(0, 13, 33000).astype(np.int64)
    max_len = 12
    x, dy, gam, off = make_inputs(dtype, lens, max_len, seed=24, base_off=1)
    dx_rows, params, ps = reference("layernorm", x, dy, gam, off, max_len)
    for mode in ("2", "0"):
        monkeypatch.setenv("ROWOP_BWD_STRIPE", mode)
        st, dxb, dgb, dbb = call(rw, "layernorm", dtype, x, dy, gam, off, max_len)
        assert st == 0 and rw.check_status() == 0
        verify("layernorm", dtype, dx_rows, params, ps, off, dxb, dgb, dbb, max_len,
               f"many rows mode {mode}")


@pytest.mark.parametrize("op", ["layernorm", "rmsnorm"])
def test_ragged_norm_backward_stripe_congruent(rw, monkeypatch, op):
    """x, dy and dx that start past a 16-byte boundary (all by the same
    amount) take the column-stripe design too: head classes count from the
    boundary before x."""
    monkeypatch.setenv("ROWOP_BWD_STRIPE", "2")
    dtype = torch.bfloat16
    lens = _ragged_lengths(dtype, 40, 25, 9000)
    max_len = int(lens.max())
    x, dy, gam, off = make_inputs(dtype, lens, max_len, seed=25)
    for shift in (3, 5):  # 6 and 10 bytes past a boundary
        st, dxb, dgb, dbb = call(rw, op, dtype, x, dy, gam, off, max_len, shift=shift)
        assert st == 0 and rw.check_status() == 0
        dx_rows, params, ps = reference(op, x, dy, gam, off, max_len)
        verify(op, dtype, dx_rows, params, ps, off, dxb, dgb, dbb, max_len,
               f"congruent {op} shift {shift}")
        assert is_canary(dxb[:G]).all() and is_canary(dxb[G + int(off[-1]):]).all()


@pytest.mark.parametrize("design", ["team", "stripe"])
def test_ragged_layernorm_backward_far_from_zero(rw, monkeypatch, design):
    """fp32 ragged LayerNorm backward of rows whose mean is 100 times their
    spread, in both designs: the stripe design's variance about each row's
    first element and its xhat = (x - mean) rstd keep the full tolerance."""
    monkeypatch.setenv("ROWOP_BWD_STRIPE", "0" if design == "team" else "2")
    dtype = torch.float32
    lens = np.array([1, 2, 9, 700, 3000, 5000, 8191, 4096, 17], dtype=np.int64)
    max_len = int(lens.max())
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    g = torch.Generator("cpu").manual_seed(31)
    x = (50.0 + 0.5 * torch.randn(int(off[-1]), generator=g, dtype=torch.float64)).float()
    dy = torch.randn(int(off[-1]), generator=g)
    gam = 1.0 + 0.2 * torch.randn(max_len, generator=g)
    st, dxb, dgb, dbb = call(rw, "layernorm", dtype, x, dy, gam, off, max_len)
    assert st == 0 and rw.check_status() == 0
    dx_rows, params, ps = reference("layernorm", x, dy, gam, off, max_len)
    verify("layernorm", dtype, dx_rows, params, ps, off, dxb, dgb, dbb, max_len,
           f"far from zero {design}")


@pytest.mark.parametrize("design", ["team", "stripe"])
@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16], ids=["f32", "bf16"])
def test_ragged_layernorm_backward_outliers(rw, monkeypatch, design, dtype):
    """Rows whose first element (or one in the middle) is an outlier 10^4
    times the spread of the rest, in both designs: statistics formed about a
    shift far from the mean would lose the variance to cancellation."""
    monkeypatch.setenv("ROWOP_BWD_STRIPE", "0" if design == "team" else "2")
    lens = np.array([5000, 3, 4096, 9000, 700, 12000], dtype=np.int64)
    max_len = int(lens.max())
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    g = torch.Generator("cpu").manual_seed(32)
    x = torch.randn(int(off[-1]), generator=g, dtype=torch.float64)
    for i, pos in enumerate((0, 0, 0, 4500, 0, 11000)):
        x[int(off[i]) + pos] = 1.0e4 if i % 2 == 0 else -3.0e3
    x, dy = x.to(dtype), torch.randn(int(off[-1]), generator=g).to(dtype)
    gam = (1.0 + 0.2 * torch.randn(max_len, generator=g)).to(dtype)
    st, dxb, dgb, dbb = call(rw, "layernorm", dtype, x, dy, gam, off, max_len)
    assert st == 0 and rw.check_status() == 0
    dx_rows, params, ps = reference("layernorm", x, dy, gam, off, max_len)
    verify("layernorm", dtype, dx_rows, params, ps, off, dxb, dgb, dbb, max_len,
           f"outliers {design} {dtype}")

