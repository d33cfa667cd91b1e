"""GPU parity of the dense entry points against the oracle, through the C ABI.

Row lengths cover the three buckets of launch_by_rows, their boundaries
(+-1 element), many tiles and ragged tails; buffers carry NaN-pattern guard
regions before and after, and the ld gaps between rows, which must come back
untouched.  Also: misaligned rows, in-place calls, determinism, and bitwise
agreement of the MEDIUM design with the cluster split at every cluster size.
"""
import os

import numpy as np
import pytest
import torch

from tests.gpu_util import (DTYPE_IDS, ALL_OPS, DTYPES, ESIZE, assert_close, canary_tensor,
                            eps_for, gen, gen_affine, is_canary, oracle_dense, to_f64)

pytestmark = pytest.mark.gpu
GUARD = 4096


@pytest.fixture(scope="module")
def rw():
    from paper_2607_23089_gb300 import build, rowop
    build.build()
    rowop.load()
    torch.cuda.set_device(0)
    return rowop


def call_dense(rw, op, x_ptr, y_ptr, g, b, rows, cols, ld, dtype, eps):
    code = rw.dtype_code(dtype)
    s = torch.cuda.current_stream().cuda_stream
    gp = g.data_ptr() if g is not None else None
    bp = b.data_ptr() if b is not None else None
    if op == "softmax":
        return rw.rowop_softmax(x_ptr, y_ptr, rows, cols, ld, code, s)
    if op == "logsoftmax":
        return rw.rowop_logsoftmax(x_ptr, y_ptr, rows, cols, ld, code, s)
    if op == "layernorm":
        return rw.rowop_layernorm(x_ptr, y_ptr, gp, bp, rows, cols, ld, code, eps, s)
    return rw.rowop_rmsnorm(x_ptr, y_ptr, gp, rows, cols, ld, code, eps, s)


def run_case(rw, op, dtype, rows, cols, ld=None, x_off=0, y_off=0, inplace=False,
             seed=0, affine=True, check=True):
    ld = ld or cols
    x = gen((rows, ld), dtype, seed)
    g, b = gen_affine(cols, dtype, seed) if (affine and op in ("layernorm", "rmsnorm")) \
        else (None, None)
    n = rows * ld
    xbuf = canary_tensor(GUARD + x_off + n + GUARD, dtype)
    xbuf[GUARD + x_off:GUARD + x_off + n] = x.reshape(-1).cuda()
    if inplace:
        ybuf, y_off = xbuf, x_off
    else:
        ybuf = canary_tensor(GUARD + y_off + n + GUARD, dtype)
    es = ESIZE[dtype]
    x_ptr = xbuf.data_ptr() + (GUARD + x_off) * es
    y_ptr = ybuf.data_ptr() + (GUARD + y_off) * es
    gd = g.cuda() if g is not None else None
    bd = b.cuda() if (b is not None and op == "layernorm") else None
    eps = eps_for(op)
    st = call_dense(rw, op, x_ptr, y_ptr, gd, bd, rows, cols, ld, dtype, eps)
    assert st == 0, rw.STATUS.get(st, st)
    torch.cuda.synchronize()
    assert rw.check_status() == 0
    y = ybuf[GUARD + y_off:GUARD + y_off + n].reshape(rows, ld)
    if check:
        ref = oracle_dense(op, x[:, :cols].double().numpy(),
                           None if gd is None else g.double().numpy(),
                           None if bd is None else b.double().numpy(), eps)
        assert_close(to_f64(y[:, :cols]), ref, dtype, f"{op} {dtype} {rows}x{cols} ld{ld}")
        # guards and ld gaps untouched
        assert is_canary(ybuf[:GUARD + y_off]).all()
        assert is_canary(ybuf[GUARD + y_off + n:]).all()
        if ld > cols and not inplace:
            assert is_canary(y[:, cols:]).all()
    return y


# row lengths: every bucket, its edges, one to many tiles, ragged tails
COLS = [1, 2, 3, 5, 8, 31, 64, 100, 128, 257, 512, 1000, 1023, 1024, 1025, 2047,
        2048, 2049, 3000, 4096, 8191, 8192, 8193, 12345, 16384, 16385, 40000,
        65539, 262144]


@pytest.mark.parametrize("dtype", DTYPES, ids=DTYPE_IDS)
@pytest.mark.parametrize("op", ALL_OPS)
@pytest.mark.parametrize("cols", COLS)
def test_dense_parity(rw, op, dtype, cols):
    rows = int(max(2, min(67, (1 << 20) // cols)))
    run_case(rw, op, dtype, rows, cols, seed=cols)


@pytest.mark.parametrize("dtype", DTYPES, ids=DTYPE_IDS)
@pytest.mark.parametrize("op", ALL_OPS)
@pytest.mark.parametrize("cols,extra,x_off,y_off", [
    (7, 1, 0, 0), (1000, 1, 1, 1), (1000, 3, 2, 0), (5000, 1, 0, 0),
    (5000, 5, 3, 3), (20000, 3, 1, 1), (20000, 1, 0, 5), (100000, 7, 3, 3)])
def test_dense_misaligned(rw, op, dtype, cols, extra, x_off, y_off):
    rows = int(max(2, min(19, (1 << 20) // cols)))
    run_case(rw, op, dtype, rows, cols, ld=cols + extra, x_off=x_off, y_off=y_off,
             seed=cols + extra)


@pytest.mark.parametrize("dtype", DTYPES, ids=DTYPE_IDS)
@pytest.mark.parametrize("op", ALL_OPS)
@pytest.mark.parametrize("cols", [100, 6000, 50000])
def test_dense_inplace(rw, op, dtype, cols):
    run_case(rw, op, dtype, 9, cols, inplace=True, seed=3 * cols)


@pytest.mark.parametrize("op", ALL_OPS)
def test_dense_without_affine(rw, op):
    for cols in (300, 9000, 70000):
        run_case(rw, op, torch.bfloat16, 5, cols, affine=False, seed=cols + 1)


@pytest.mark.parametrize("op", ALL_OPS)
def test_dense_deterministic(rw, op):
    for cols in (777, 7777, 77777):
        a = run_case(rw, op, torch.float32, 6, cols, seed=11, check=False).clone()
        b = run_case(rw, op, torch.float32, 6, cols, seed=11, check=False)
        assert torch.equal(a.view(torch.int32), b.view(torch.int32))


KNOBS = ("ROWOP_FORCE_BUCKET", "ROWOP_CLUSTER", "ROWOP_GROUP_WARPS", "ROWOP_STAGES")


def _forced(rw, op, dtype, rows, cols, bucket, cluster=None, ld=None, x_off=0,
            group_warps=None, stages=None):
    old = {k: os.environ.get(k) for k in KNOBS}
    try:
        os.environ["ROWOP_FORCE_BUCKET"] = str(bucket)
        for k, v in (("ROWOP_CLUSTER", cluster), ("ROWOP_GROUP_WARPS", group_warps),
                     ("ROWOP_STAGES", stages)):
            if v:
                os.environ[k] = str(v)
            else:
                os.environ.pop(k, None)
        return run_case(rw, op, dtype, rows, cols, ld=ld, x_off=x_off, y_off=x_off,
                        seed=cols).clone()
    finally:
        for k, v in old.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v


def _bits(t):
    return t.view(torch.int32) if t.dtype == torch.float32 else t.view(torch.int16)


@pytest.mark.parametrize("dtype", DTYPES, ids=DTYPE_IDS)
@pytest.mark.parametrize("op", ALL_OPS)
@pytest.mark.parametrize("cols,ld,x_off", [(900, None, 0), (6000, None, 0),
                                          (6000, 6003, 1), (40000, None, 0),
                                          (40001, 40005, 3)])
def test_forced_designs_agree(rw, op, dtype, cols, ld, x_off):
    """Every bucket design is correct on the same rows, and the MEDIUM design
    and the cluster split (any cluster size) agree bit for bit."""
    rows = 5
    medium = _forced(rw, op, dtype, rows, cols, 1, ld=ld, x_off=x_off)
    for cs in (2, 4, 8, 16):
        large = _forced(rw, op, dtype, rows, cols, 2, cluster=cs, ld=ld, x_off=x_off)
        assert torch.equal(_bits(medium), _bits(large)), f"cluster {cs}"
    if cols * ESIZE[dtype] <= 4096 + 512:
        _forced(rw, op, dtype, rows, cols, 0, ld=ld, x_off=x_off)


@pytest.mark.parametrize("dtype", DTYPES, ids=DTYPE_IDS)
@pytest.mark.parametrize("op", ALL_OPS)
@pytest.mark.parametrize("cols,ld,x_off", [(3000, None, 0), (6000, 6003, 1),
                                          (40001, 40005, 3)])
def test_group_sizes_agree(rw, op, dtype, cols, ld, x_off):
    """The tile kernel's consumer warps work in groups of W (1, 2, 4 or 8
    warps per item, several items at once).  Which warp reduces which tile
    does not change the arithmetic: every W, with few or many stages, gives
    the same bits, in the one-CTA design and in the cluster split.  37 rows
    give every group several items and a partial last round."""
    rows = 37
    ref = _forced(rw, op, dtype, rows, cols, 1, ld=ld, x_off=x_off, group_warps=8)
    for w in (1, 2, 4):
        for stages in (None, 8 // w):
            got = _forced(rw, op, dtype, rows, cols, 1, ld=ld, x_off=x_off, group_warps=w,
                          stages=stages)
            assert torch.equal(_bits(ref), _bits(got)), f"MEDIUM W={w} stages={stages}"
    for cs, w in ((2, 1), (4, 2), (8, 4)):
        got = _forced(rw, op, dtype, rows, cols, 2, cluster=cs, ld=ld, x_off=x_off,
                      group_warps=w)
        assert torch.equal(_bits(ref), _bits(got)), f"cluster {cs} W={w}"


@pytest.mark.parametrize("dtype", DTYPES, ids=DTYPE_IDS)
@pytest.mark.parametrize("op", ["softmax", "logsoftmax"])
@pytest.mark.parametrize("cols", [1, 5, 64, 255, 1000, 2047, 3000, 8192, 20000, 70001])
def test_online_softmax_variant(rw, op, dtype, cols, monkeypatch):
    """The one-pass (online) softmax statistics, selected by
    ROWOP_SOFTMAX_ONLINE -- a running maximum in the SMALL design, one sweep
    over each staged tile in the MEDIUM / LARGE designs -- meet the same
    tolerance against the oracle, also on rows whose maximum arrives late and
    rows with -inf entries."""
    monkeypatch.setenv("ROWOP_SOFTMAX_ONLINE", "1")
    run_case(rw, op, dtype, 37, cols, seed=cols + 3)
    rows = 6
    x = torch.linspace(-20, 20, cols).repeat(rows, 1)  # increasing: the maximum is last
    x[1] = x[1].flip(0)
    x[2, ::3] = -float("inf")
    x = x.to(dtype)
    y = rw.run(op, x.cuda()).cpu()
    ref = oracle_dense(op, x.double().numpy())
    assert_close(to_f64(y), ref, dtype, f"online {op}")


@pytest.mark.parametrize("op", ["softmax", "logsoftmax"])
@pytest.mark.parametrize("cs", [2, 8, 16])
def test_online_softmax_cluster(rw, op, cs, monkeypatch):
    """The online tile statistics across a cluster split of every size."""
    monkeypatch.setenv("ROWOP_SOFTMAX_ONLINE", "1")
    monkeypatch.setenv("ROWOP_FORCE_BUCKET", "2")
    monkeypatch.setenv("ROWOP_CLUSTER", str(cs))
    for dtype in (torch.float32, torch.bfloat16):
        run_case(rw, op, dtype, 5, 50001, seed=cs)
