"""GPU parity of the fused residual add + LayerNorm / RMSNorm, through the C
ABI.  The stored sum must equal the oracle's sum rounded to the I/O type bit
for bit, the normalised output must match the oracle's norm of that stored
sum within the tolerance, and -- since the fused kernels reduce and normalise
the stored sum with the same code as the plain norms -- it must also equal,
bit for bit, the plain norm run on the sum.  Covers every bucket design,
misaligned rows, strided rows, residual rows at another alignment, and the
residual stream updated in place."""
import numpy as np
import pytest
import torch

from oracle import rowop_oracle as orc
from tests.gpu_util import (DTYPE_IDS, DTYPES, ESIZE, assert_close, canary_tensor, gen_affine,
                            is_canary, to_f64)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def rw():
    from paper_2607_23089_gb300 import build, rowop
    build.build()
    rowop.load()
    torch.cuda.set_device(0)
    return rowop


def _bits(t):
    return t.view(torch.int32) if t.dtype == torch.float32 else t.view(torch.int16)


def _buf(rows, ld, dtype, off, fill=None):
    G = 64
    b = canary_tensor(G + off + rows * ld + G, dtype)
    if fill is not None:
        b[G + off:G + off + rows * ld] = fill.reshape(-1).cuda()
    return b, G + off


def run(rw, op, dtype, rows, cols, ld=None, offs=(0, 0, 0, 0), inplace=None, seed=0,
        affine=True):
    ld = ld or cols
    g = torch.Generator("cpu").manual_seed(seed)
    x = (2 * torch.randn(rows, ld, generator=g)).to(dtype)
    r = (torch.randn(rows, ld, generator=g) + 0.5).to(dtype)
    gam, bet = gen_affine(cols, dtype, seed) if affine else (None, None)
    es = ESIZE[dtype]
    xb, xo = _buf(rows, ld, dtype, offs[0], x)
    rb, ro = _buf(rows, ld, dtype, offs[1], r)
    yb, yo = _buf(rows, ld, dtype, offs[3])
    if inplace == "x":
        sb, so = xb, xo
    elif inplace == "r":
        sb, so = rb, ro
    else:
        sb, so = _buf(rows, ld, dtype, offs[2])
    p = lambda b, o: b.data_ptr() + o * es  # noqa: E731
    gd = gam.cuda() if gam is not None else None
    bd = bet.cuda() if bet is not None else None
    stream = torch.cuda.current_stream().cuda_stream
    eps = 1e-5 if op == "layernorm" else 1e-6
    code = rw.dtype_code(dtype)
    if op == "layernorm":
        st = rw.rowop_add_layernorm(p(xb, xo), p(rb, ro), p(sb, so), p(yb, yo),
                                    gd.data_ptr() if gd is not None else None,
                                    bd.data_ptr() if bd is not None else None,
                                    rows, cols, ld, code, eps, stream)
    else:
        st = rw.rowop_add_rmsnorm(p(xb, xo), p(rb, ro), p(sb, so), p(yb, yo),
                                  gd.data_ptr() if gd is not None else None,
                                  rows, cols, ld, code, eps, stream)
    assert st == 0, rw.STATUS.get(st, st)
    torch.cuda.synchronize()
    view = lambda b, o: b[o:o + rows * ld].reshape(rows, ld)  # noqa: E731
    s = view(sb, so)
    y = view(yb, yo)
    x64 = x[:, :cols].double().numpy()
    r64 = r[:, :cols].double().numpy()
    if op == "layernorm":
        s_ref, y_ref = orc.add_layernorm(x64, r64, dtype, gam.double().numpy() if affine else None,
                                         bet.double().numpy() if affine else None, eps=eps)
    else:
        s_ref, y_ref = orc.add_rmsnorm(x64, r64, dtype, gam.double().numpy() if affine else None,
                                       eps=eps)
    # the stored sum, bit for bit; the normalised rows within the tolerance
    s_want = torch.from_numpy(s_ref).to(dtype)
    assert torch.equal(_bits(s[:, :cols].cpu()), _bits(s_want))
    assert_close(to_f64(y[:, :cols]), y_ref, dtype, f"add_{op} {dtype}")
    # nothing outside the rows' columns was written
    if ld > cols:
        assert is_canary(y[:, cols:]).all()
        if inplace is None:
            assert is_canary(s[:, cols:]).all()
    # the fused output is the plain norm of the stored sum, bit for bit
    s_copy = s[:, :cols].contiguous()
    if op == "layernorm":
        plain = rw.layernorm(s_copy, gd, bd, eps)
    else:
        plain = rw.rmsnorm(s_copy, gd, eps)
    return y[:, :cols], plain


COLS = [1, 100, 1000, 2048, 3000, 6000, 40000]


@pytest.mark.parametrize("dtype", DTYPES, ids=DTYPE_IDS)
@pytest.mark.parametrize("op", ["layernorm", "rmsnorm"])
@pytest.mark.parametrize("cols", COLS)
def test_add_norm_parity(rw, op, dtype, cols):
    rows = 7 if cols > 10000 else 33
    y, plain = run(rw, op, dtype, rows, cols, seed=cols)
    if ESIZE[dtype] * cols > 4096:  # the tile designs reduce the stored sum exactly as the plain norm
        assert torch.equal(_bits(y), _bits(plain))


@pytest.mark.parametrize("dtype", DTYPES, ids=DTYPE_IDS)
@pytest.mark.parametrize("op", ["layernorm", "rmsnorm"])
@pytest.mark.parametrize("cols,ld,offs", [(3001, 3011, (1, 1, 1, 5)), (777, 800, (0, 3, 3, 0)),
                                          (9000, 9005, (2, 7, 5, 1)), (1000, 1003, (3, 3, 3, 3))])
def test_add_norm_misaligned(rw, op, dtype, cols, ld, offs):
    run(rw, op, dtype, 9, cols, ld=ld, offs=offs, seed=cols + ld)


@pytest.mark.parametrize("op", ["layernorm", "rmsnorm"])
@pytest.mark.parametrize("where", ["x", "r"])
@pytest.mark.parametrize("cols", [500, 6000, 70000])
def test_add_norm_inplace(rw, op, where, cols):
    run(rw, op, torch.bfloat16, 5, cols, inplace=where, seed=3)


def test_add_norm_no_affine(rw):
    for op in ("layernorm", "rmsnorm"):
        for cols in (200, 5000):
            run(rw, op, torch.float32, 6, cols, affine=False, seed=9)


@pytest.mark.parametrize("op", ["layernorm", "rmsnorm"])
def test_add_norm_designs_agree(rw, op, monkeypatch):
    """The one-CTA design and the cluster split at several cluster sizes
    give the same bits on the fused residual path too."""
    outs = []
    for bucket, cs in ((1, None), (2, 2), (2, 4), (2, 16)):
        monkeypatch.setenv("ROWOP_FORCE_BUCKET", str(bucket))
        if cs:
            monkeypatch.setenv("ROWOP_CLUSTER", str(cs))
        else:
            monkeypatch.delenv("ROWOP_CLUSTER", raising=False)
        y, _ = run(rw, op, torch.float32, 5, 40001, seed=21)
        outs.append(y.clone())
    for o in outs[1:]:
        assert torch.equal(_bits(outs[0]), _bits(o))


def test_add_norm_argument_checks(rw):
    x = torch.zeros(4, 8, device="cuda")
    st = rw.rowop_add_rmsnorm(x.data_ptr(), None, x.data_ptr(), x.data_ptr(), None, 4, 8, 8,
                              rw.ROWOP_F32, 1e-6, None)
    assert st == rw.ROWOP_ERR_INVALID_ARG
    st = rw.rowop_add_layernorm(x.data_ptr(), x.data_ptr(), None, x.data_ptr(), None, None,
                                4, 8, 8, rw.ROWOP_F32, 1e-5, None)
    assert st == rw.ROWOP_ERR_INVALID_ARG
