"""GPU parity of the ragged (CSR-offset) entry points, through the C ABI.

One call mixes rows of every bucket (empty, length 1, SMALL, MEDIUM and
cluster-split LARGE rows).  Checks: values against the oracle; the bucket
every row was dispatched to (read back from the workspace) equals the
dispatch rule exactly; a ragged row equals, bit for bit, a dense call on the
same row at the same 16-byte alignment; rejected rows (decreasing offsets,
len > max_len) are left untouched and flagged; in-place calls.
"""
import numpy as np
import pytest
import torch

from oracle import rowop_oracle as orc
from tests.gpu_util import (DTYPE_IDS, ALL_OPS, DTYPES, ESIZE, assert_close, canary_tensor,
                            eps_for, gen_affine, is_canary, oracle_ragged, to_f64)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def rw():
    from paper_2607_23089_gb300 import build, rowop
    build.build()
    rowop.load()
    torch.cuda.set_device(0)
    return rowop


def mixed_lengths(dtype, rows, seed, max_len):
    """Lengths spread over all buckets, with empty and length-1 rows."""
    es = ESIZE[dtype]
    g = np.random.default_rng(seed)
    small = 4096 // es
    med = 32768 // es
    pools = [(0, 2), (1, 64), (65, small), (small + 1, med), (med + 1, max_len)]
    lens = []
    for i in range(rows):
        lo, hi = pools[i % len(pools)]
        hi = max(lo, min(hi, max_len))
        lens.append(int(g.integers(lo, hi + 1)))
    lens = np.array(lens, dtype=np.int64)
    g.shuffle(lens)
    return lens


def call_ragged(rw, op, x, y, off, rows, max_len, g, b, dtype, eps, ws):
    code = rw.dtype_code(dtype)
    s = torch.cuda.current_stream().cuda_stream
    gp = None if g is None else g.data_ptr()
    bp = None if b is None else b.data_ptr()
    if op == "softmax":
        return rw.rowop_softmax_ragged(x, y, off, rows, max_len, code, ws.data_ptr(),
                                       ws.numel(), s)
    if op == "logsoftmax":
        return rw.rowop_logsoftmax_ragged(x, y, off, rows, max_len, code, ws.data_ptr(),
                                          ws.numel(), s)
    if op == "layernorm":
        return rw.rowop_layernorm_ragged(x, y, gp, bp, off, rows, max_len, code, eps,
                                         ws.data_ptr(), ws.numel(), s)
    return rw.rowop_rmsnorm_ragged(x, y, gp, off, rows, max_len, code, eps,
                                   ws.data_ptr(), ws.numel(), s)


def run_ragged(rw, op, dtype, lens, max_len, seed, base_off=0, inplace=False,
               offsets=None):
    off = offsets if offsets is not None else \
        np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    total = max(int(off.max()), 1)
    rows = off.shape[0] - 1
    gx = torch.Generator("cpu").manual_seed(seed)
    x = (3.0 * torch.randn(total, generator=gx)).to(dtype)
    gam, bet = gen_affine(max(max_len, 1), dtype, seed)
    G = 256
    xbuf = canary_tensor(G + base_off + total + G, dtype)
    xbuf[G + base_off:G + base_off + total] = x.cuda()
    ybuf = xbuf if inplace else canary_tensor(G + base_off + total + G, dtype)
    es = ESIZE[dtype]
    xp = xbuf.data_ptr() + (G + base_off) * es
    yp = ybuf.data_ptr() + (G + base_off) * es
    offd = torch.from_numpy(off).cuda()
    ws = rw.ragged_workspace(rows)
    gd = gam.cuda() if op in ("layernorm", "rmsnorm") else None
    bd = bet.cuda() if op == "layernorm" else None
    eps = eps_for(op)
    st = call_ragged(rw, op, xp, yp, offd.data_ptr(), rows, max_len, gd, bd, dtype, eps, ws)
    assert st == 0, rw.STATUS.get(st, st)
    torch.cuda.synchronize()
    y = ybuf[G + base_off:G + base_off + total]
    return dict(x=x, y=y, ybuf=ybuf, off=off, ws=ws, gam=gam, bet=bet, eps=eps,
                G=G, base_off=base_off, total=total)


@pytest.mark.parametrize("dtype", DTYPES, ids=DTYPE_IDS)
@pytest.mark.parametrize("op", ALL_OPS)
@pytest.mark.parametrize("base_off", [0, 3])
def test_ragged_parity(rw, op, dtype, base_off):
    max_len = 70000 if dtype == torch.float32 else 40000
    lens = mixed_lengths(dtype, 160, seed=5 + base_off, max_len=max_len)
    r = run_ragged(rw, op, dtype, lens, max_len, seed=17 + base_off, base_off=base_off)
    assert rw.check_status() == 0
    ref = oracle_ragged(op, r["x"].double().numpy(), r["off"],
                        r["gam"].double().numpy(), r["bet"].double().numpy(), r["eps"])
    assert_close(to_f64(r["y"]), ref, dtype, f"ragged {op} {dtype}")
    G, b = r["G"], r["base_off"]
    assert is_canary(r["ybuf"][:G + b]).all()
    assert is_canary(r["ybuf"][G + b + r["total"]:]).all()
    # dispatch: the bucket byte of every row equals the rule, bit for bit
    rows = len(lens)
    buckets = r["ws"][256:256 + rows].cpu().numpy()
    want = np.array([orc.bucket(int(n), ESIZE[dtype]) for n in lens], dtype=np.uint8)
    assert (buckets == want).all()
    assert r["ws"][:4].view(torch.int32).item() == 0


@pytest.mark.parametrize("dtype", DTYPES, ids=DTYPE_IDS)
@pytest.mark.parametrize("op", ALL_OPS)
def test_ragged_row_equals_dense_row(rw, op, dtype):
    """A ragged row and a dense call on the same row at the same 16-byte
    alignment give identical bits."""
    max_len = 50000 if dtype == torch.float32 else 30000
    lens = mixed_lengths(dtype, 40, seed=9, max_len=max_len)
    r = run_ragged(rw, op, dtype, lens, max_len, seed=23, base_off=1)
    es = ESIZE[dtype]
    code = rw.dtype_code(dtype)
    s = torch.cuda.current_stream().cuda_stream
    gd = r["gam"].cuda()
    bd = r["bet"].cuda()
    for i in range(len(lens)):
        n = int(lens[i])
        if n == 0:
            continue
        start = int(r["off"][i]) + r["base_off"]  # element index in the guarded buffer
        h = (start * es) % 16 // es
        buf = canary_tensor(64 + h + n + 64, dtype)
        buf[64 + h:64 + h + n] = r["x"][r["off"][i]:r["off"][i] + n].cuda()
        out = canary_tensor(64 + h + n + 64, dtype)
        xp = buf.data_ptr() + (64 + h) * es
        yp = out.data_ptr() + (64 + h) * es
        if op == "softmax":
            st = rw.rowop_softmax(xp, yp, 1, n, n, code, s)
        elif op == "logsoftmax":
            st = rw.rowop_logsoftmax(xp, yp, 1, n, n, code, s)
        elif op == "layernorm":
            st = rw.rowop_layernorm(xp, yp, gd.data_ptr(), bd.data_ptr(), 1, n, n, code,
                                    r["eps"], s)
        else:
            st = rw.rowop_rmsnorm(xp, yp, gd.data_ptr(), 1, n, n, code, r["eps"], s)
        assert st == 0
        dense = out[64 + h:64 + h + n]
        rag = r["y"][r["off"][i]:r["off"][i] + n]
        bits = (lambda t: t.view(torch.int32)) if dtype == torch.float32 else \
            (lambda t: t.view(torch.int16))
        assert torch.equal(bits(dense), bits(rag)), f"row {i} len {n}"


@pytest.mark.parametrize("op", ALL_OPS)
def test_ragged_inplace(rw, op):
    dtype = torch.bfloat16
    lens = mixed_lengths(dtype, 50, seed=31, max_len=30000)
    x0 = None
    r = run_ragged(rw, op, dtype, lens, 30000, seed=41, base_off=5, inplace=True)
    ref = oracle_ragged(op, r["x"].double().numpy(), r["off"], r["gam"].double().numpy(),
                        r["bet"].double().numpy(), r["eps"])
    assert_close(to_f64(r["y"]), ref, dtype, f"ragged in-place {op}")
    del x0


def test_ragged_rejects_bad_rows(rw):
    dtype = torch.float32
    # row 0 runs backwards (negative length), row 6 is longer than max_len;
    # the legal rows in between do not overlap anything.
    off = np.array([50, 10, 60, 360, 9360, 9380, 9480, 9480 + 9500], dtype=np.int64)
    max_len = 9100
    r = run_ragged(rw, "softmax", dtype, None, max_len, seed=3, offsets=off)
    st = rw.check_status()
    assert st == rw.ROWOP_ERR_BAD_OFFSETS
    assert rw.check_status() == 0  # the status word was cleared
    rows = off.shape[0] - 1
    buckets = r["ws"][256:256 + rows].cpu().numpy()
    lens_eff = np.diff(off)
    for i in range(rows):
        n = int(lens_eff[i])
        seg = r["y"][int(off[i]):int(off[i]) + max(n, 0)]
        if n < 0 or n > max_len:
            assert buckets[i] == 255
            if n > 0:
                assert is_canary(seg).all()
        else:
            assert buckets[i] == orc.bucket(n, 4)
            ref = orc.softmax(r["x"][int(off[i]):int(off[i]) + n].double().numpy()[None])[0]
            assert_close(to_f64(seg), ref, dtype, f"row {i}")
    assert r["ws"][:4].view(torch.int32).item() == 2


def test_ragged_all_empty_and_tiny(rw):
    for lens in ([0, 0, 0], [1], [1, 0, 1, 2]):
        lens = np.array(lens, dtype=np.int64)
        r = run_ragged(rw, "logsoftmax", torch.float32, lens, 4, seed=1)
        assert rw.check_status() == 0
        covered = int(r["off"][-1])
        if covered == 0:
            assert is_canary(r["y"]).all()  # nothing to write
            continue
        ref = oracle_ragged("logsoftmax", r["x"][:covered].double().numpy(), r["off"])
        assert_close(to_f64(r["y"][:covered]), ref, torch.float32, "tiny")


@pytest.mark.parametrize("dtype", DTYPES, ids=DTYPE_IDS)
@pytest.mark.parametrize("op", ("softmax", "layernorm"))
def test_ragged_group_sizes_agree(rw, op, dtype, monkeypatch):
    """The fused ragged kernel gives the same bits whatever the consumer
    group size (W warps per item) and cluster size it runs with."""
    max_len = 70000 if dtype == torch.float32 else 40000
    lens = mixed_lengths(dtype, 300, seed=41, max_len=max_len)
    ref = run_ragged(rw, op, dtype, lens, max_len, seed=43, base_off=1)["y"].clone()
    bits = (lambda t: t.view(torch.int32)) if dtype == torch.float32 else \
        (lambda t: t.view(torch.int16))
    for w, cs in ((1, None), (2, 4), (4, None), (8, 2)):
        monkeypatch.setenv("ROWOP_GROUP_WARPS", str(w))
        if cs:
            monkeypatch.setenv("ROWOP_CLUSTER", str(cs))
        else:
            monkeypatch.delenv("ROWOP_CLUSTER", raising=False)
        got = run_ragged(rw, op, dtype, lens, max_len, seed=43, base_off=1)["y"]
        assert rw.check_status() == 0
        assert torch.equal(bits(ref), bits(got)), f"W={w} cluster={cs}"


@pytest.mark.parametrize("rows", [1025, 5000, 300000])
def test_ragged_many_classify_blocks(rw, rows):
    """Enough rows for several classify blocks (1024 rows each, at most 256
    blocks): every block lists its own rows and the fused kernel maps list
    positions across blocks.  Rows of every bucket sit in different blocks,
    some rejected; values, dispatch bytes and the status all check out."""
    dtype = torch.bfloat16
    op = "layernorm"
    g = np.random.default_rng(rows)
    max_len = 20000
    lens = g.integers(0, 40, size=rows)
    lens[::997] = 3000      # MEDIUM
    lens[5::1999] = 19000   # LARGE
    lens[7::2503] = 0
    r = run_ragged(rw, op, dtype, lens, max_len, seed=rows % 97)
    assert rw.check_status() == 0
    ref = oracle_ragged(op, r["x"].double().numpy(), r["off"], r["gam"].double().numpy(),
                        r["bet"].double().numpy(), r["eps"])
    assert_close(to_f64(r["y"]), ref, dtype, f"ragged {rows} rows")
    buckets = r["ws"][256:256 + rows].cpu().numpy()
    want = np.array([orc.bucket(int(n), ESIZE[dtype]) for n in lens], dtype=np.uint8)
    assert (buckets == want).all()


def test_ragged_bad_rows_in_several_blocks(rw):
    """Rejected rows in different classify blocks all raise the status bit of
    the call and are skipped; the others are normalised."""
    dtype = torch.float32
    rows = 3000
    g = np.random.default_rng(3)
    lens = g.integers(1, 300, size=rows)
    bad = [10, 1500, 2990]
    lens[bad] = 500  # longer than max_len
    r = run_ragged(rw, "softmax", dtype, lens, 400, seed=5)
    assert rw.check_status() == rw.ROWOP_ERR_BAD_OFFSETS
    buckets = r["ws"][256:256 + rows].cpu().numpy()
    assert all(buckets[i] == 255 for i in bad)
    assert r["ws"][:4].view(torch.int32).item() == 2
    off = r["off"]
    for i in bad:
        assert is_canary(r["y"][int(off[i]):int(off[i + 1])]).all()
    good = np.ones(rows, dtype=bool)
    good[bad] = False
    for i in np.flatnonzero(good)[::97]:
        seg = r["y"][int(off[i]):int(off[i + 1])]
        ref = orc.softmax(r["x"][int(off[i]):int(off[i + 1])].double().numpy()[None])[0]
        assert_close(to_f64(seg), ref, dtype, f"row {i}")


@pytest.mark.parametrize("op", ALL_OPS)
def test_ragged_chunked_calls_equal_one_call(rw, op):
    """Rows are independent: calls over contiguous chunks of rows, each given
    its slice of the offsets (a first offset other than 0), write bitwise what
    one call over all rows writes -- the decomposition the benchmark's
    end-to-end pipeline uses."""
    dtype = torch.bfloat16
    max_len = 20000
    lens = mixed_lengths(dtype, 90, 31, max_len)
    whole = run_ragged(rw, op, dtype, lens, max_len, seed=31)
    off = whole["off"]
    offd = torch.from_numpy(off).cuda()
    es = ESIZE[dtype]
    G = whole["G"]
    ybuf = canary_tensor(G + whole["total"] + G, dtype)
    xbuf = canary_tensor(G + whole["total"] + G, dtype)
    xbuf[G:G + whole["total"]] = whole["x"].cuda()
    gd = whole["gam"].cuda() if op in ("layernorm", "rmsnorm") else None
    bd = whole["bet"].cuda() if op == "layernorm" else None
    bounds = [0, 1, 17, 40, 41, 90]
    for r0, r1 in zip(bounds[:-1], bounds[1:]):
        ws = rw.ragged_workspace(r1 - r0)
        st = call_ragged(rw, op, xbuf.data_ptr() + G * es, ybuf.data_ptr() + G * es,
                         offd.data_ptr() + 8 * r0, r1 - r0, max_len, gd, bd, dtype,
                         whole["eps"], ws)
        assert st == 0, rw.STATUS.get(st, st)
    torch.cuda.synchronize()
    got = ybuf[G:G + whole["total"]]
    assert torch.equal(got.view(torch.int16), whole["y"].view(torch.int16))


@pytest.mark.parametrize("op", ["softmax", "layernorm"])
def test_planned_call_refuses_a_mismatched_plan(rw, op):
    """A plan made for another element type, or for a longer max_len, than the
    planned call that reuses it: the rows whose record does not fit the call
    (another bucket for the call's element size, or longer than its max_len)
    are skipped, left untouched, and flagged as rejected rows; the others are
    computed as usual."""
    s = torch.cuda.current_stream().cuda_stream
    # lengths as a bf16 plan sorts them: SMALL, SMALL (a MEDIUM row in fp32),
    # MEDIUM, MEDIUM (a LARGE row in fp32), LARGE, LARGE
    lens = np.array([100, 1500, 3000, 10000, 20000, 25000], dtype=np.int64)
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    rows, total = len(lens), int(off[-1])
    offd = torch.from_numpy(off).cuda()
    gx = torch.Generator("cpu").manual_seed(61)
    x = (3.0 * torch.randn(total, generator=gx)).float()
    gam, bet = gen_affine(30000, torch.float32, 61)
    gd, bd = gam.cuda(), bet.cuda()
    eps = eps_for(op)
    ws = rw.ragged_workspace(rows)

    params = {torch.float32: (gd, bd), torch.bfloat16: (gd.bfloat16(), bd.bfloat16())}

    def planned(dtype, max_len):
        xd = x.to(dtype).cuda()
        y = canary_tensor(total, dtype)
        code = rw.dtype_code(dtype)
        gp, bp = params[dtype]  # kept alive until the call has run
        if op == "softmax":
            st = rw.rowop_softmax_ragged_planned(xd.data_ptr(), y.data_ptr(), offd.data_ptr(),
                                                 rows, max_len, code, ws.data_ptr(), ws.numel(), s)
        else:
            st = rw.rowop_layernorm_ragged_planned(xd.data_ptr(), y.data_ptr(), gp.data_ptr(),
                                                   bp.data_ptr(), offd.data_ptr(), rows, max_len,
                                                   code, eps, ws.data_ptr(), ws.numel(), s)
        assert st == rw.ROWOP_OK
        torch.cuda.synchronize()
        return xd, y

    def check(dtype, xd, y, skipped):
        assert rw.check_status() == rw.ROWOP_ERR_BAD_OFFSETS
        ref = oracle_ragged(op, xd.double().cpu().numpy(), off,
                            gam.to(dtype).double().numpy(), bet.to(dtype).double().numpy(), eps)
        for i in range(rows):
            seg = slice(int(off[i]), int(off[i + 1]))
            if i in skipped:
                assert is_canary(y[seg]).all(), f"row {i} written"
            else:
                assert_close(to_f64(y[seg]), ref[seg], dtype, f"row {i}")

    # a bf16 plan reused by an fp32 call
    st = rw.rowop_ragged_plan(offd.data_ptr(), rows, 30000, rw.ROWOP_BF16, ws.data_ptr(),
                              ws.numel(), s)
    assert st == rw.ROWOP_OK
    xd, y = planned(torch.float32, 30000)
    check(torch.float32, xd, y, {1, 3})
    # a plan for max_len 30000 reused by a call whose max_len is 22000
    xd, y = planned(torch.bfloat16, 22000)
    check(torch.bfloat16, xd, y, {5})
    # the matching call still works on the same plan
    xd, y = planned(torch.bfloat16, 30000)
    assert rw.check_status() == rw.ROWOP_OK
    ref = oracle_ragged(op, xd.double().cpu().numpy(), off,
                        gam.to(torch.bfloat16).double().numpy(),
                        bet.to(torch.bfloat16).double().numpy(), eps)
    assert_close(to_f64(y), ref, torch.bfloat16, "matching plan")


@pytest.mark.parametrize("dtype", DTYPES, ids=DTYPE_IDS)
@pytest.mark.parametrize("op", ALL_OPS)
@pytest.mark.parametrize("base_off", [0, 1, 5])
def test_ragged_longest_and_boundary_rows(rw, op, dtype, base_off):
    """Rows at the bucket boundaries (+-1 element), the longest rows the call
    allows at several head offsets (so their last chunk may start a tile of
    its own), one- to three-element rows, among rows of every bucket."""
    es = ESIZE[dtype]
    max_len = 32768 if es == 2 else 40000
    med = 32768 // es
    special = [max_len, max_len - 1, max_len - 7, med, med + 1, med - 1, med + 9, 4096 // es,
               4096 // es + 1, 1, 2, 3, 512 * 16 // es, 512 * 16 // es + 1]
    lens = np.concatenate([np.array(special, dtype=np.int64),
                           mixed_lengths(dtype, 120, seed=base_off + 101, max_len=max_len)])
    np.random.default_rng(7).shuffle(lens)
    got = run_ragged(rw, op, dtype, lens, max_len, seed=77, base_off=base_off)
    assert rw.check_status() == 0
    ref = oracle_ragged(op, got["x"].double().numpy(), got["off"], got["gam"].double().numpy(),
                        got["bet"].double().numpy(), got["eps"])
    assert_close(to_f64(got["y"]), ref, dtype, f"{op} boundary rows")
    G, b = got["G"], got["base_off"]
    assert is_canary(got["ybuf"][:G + b]).all()
    assert is_canary(got["ybuf"][G + b + got["total"]:]).all()
