"""GPU parity of the Hyena FFT-size padding and the MoE group score, through
the C ABI, against the double-precision oracle.

fp32 padding is compared bit for bit: the product of two float32 values is
exact in double, so the oracle's value rounded to float32 is the correctly
rounded product the GPU forms.  bf16 padding rounds that fp32 product once
more and is held to its tolerance (so is fp16).  The group score is compared bit for
bit in every dtype: the sum of the two largest scores is exact in double and
the GPU rounds it to float32 once.
"""
import numpy as np
import pytest
import torch

from oracle import rowop_oracle as orc
from tests.gpu_util import DTYPE_IDS, DTYPES, ESIZE, assert_close, canary_tensor, is_canary, to_f64

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


def run_pad(rw, dtype, rows, seqlen, fft, scale, ld_in=None, ld_out=None, off_in=0,
            off_out=0, seed=0):
    ld_in = ld_in or max(seqlen, 1)
    ld_out = ld_out or fft
    g = torch.Generator("cpu").manual_seed(seed)
    x = (3 * torch.randn(rows, ld_in, generator=g)).to(dtype)
    es = ESIZE[dtype]
    G = 64
    xbuf = canary_tensor(G + off_in + rows * ld_in + G, dtype)
    xbuf[G + off_in:G + off_in + rows * ld_in] = x.reshape(-1).cuda()
    ybuf = canary_tensor(G + off_out + rows * ld_out + G, dtype)
    xp = xbuf.data_ptr() + (G + off_in) * es
    yp = ybuf.data_ptr() + (G + off_out) * es
    st = rw.rowop_pad_scale(xp if seqlen > 0 else None, yp, rows, seqlen, fft, ld_in, ld_out,
                            scale, rw.dtype_code(dtype), torch.cuda.current_stream().cuda_stream)
    assert st == 0, rw.STATUS.get(st, st)
    torch.cuda.synchronize()
    y = ybuf[G + off_out:G + off_out + rows * ld_out].reshape(rows, ld_out)
    ref = orc.pad_scale(x[:, :seqlen].double().numpy(), fft, scale)
    # guards and the columns past fft_size are untouched
    assert is_canary(ybuf[:G + off_out]).all()
    assert is_canary(ybuf[G + off_out + rows * ld_out:]).all()
    if ld_out > fft:
        assert is_canary(y[:, fft:]).all()
    return y[:, :fft], ref


PAD_CASES = [
    (5, 3000, 4096, 0.25, None, None, 0, 0),      # vector path, boundary chunk inside a segment
    (3, 4096, 4096, -1.5, None, None, 0, 0),      # no padding at all
    (4, 0, 256, 2.0, None, None, 0, 0),           # all zeros, no input
    (9, 1000, 2050, 0.5, None, None, 0, 0),       # fft not a whole number of chunks: element path
    (6, 777, 5000, 0.125, 800, 5008, 0, 0),       # strided rows
    (5, 640, 1280, 3.0, None, None, 1, 3),        # misaligned bases: element path
    (70000, 7, 16, 1.0, None, None, 0, 0),        # many short rows: every warp loops
    (2, 12000, 40000, 0.001, None, None, 0, 0),   # several segments per row
]


@pytest.mark.parametrize("dtype", DTYPES, ids=DTYPE_IDS)
@pytest.mark.parametrize("case", PAD_CASES, ids=lambda c: f"{c[0]}x{c[1]}->{c[2]}")
def test_pad_scale_parity(rw, dtype, case):
    rows, seqlen, fft, scale, ld_in, ld_out, off_in, off_out = case
    y, ref = run_pad(rw, dtype, rows, seqlen, fft, scale, ld_in, ld_out, off_in, off_out,
                     seed=rows + seqlen)
    # the zero tail is exact in every dtype
    assert (y[:, seqlen:].float() == 0).all()
    if dtype == torch.float32:
        want = torch.from_numpy(ref.astype(np.float32))
        assert torch.equal(_bits(y.cpu()), _bits(want))
    else:
        assert_close(to_f64(y), ref, dtype, f"pad_scale {dtype}")


def test_pad_scale_workload_sampled(rw):
    from paper_2607_23089_gb300 import workloads as wl
    case = wl.hyena_pad()
    x = case.x.cuda()
    y = rw.pad_scale(x, case.meta["fft_size"], case.meta["scale"])
    torch.cuda.synchronize()
    idx = np.random.default_rng(1).choice(x.shape[0], 64, replace=False)
    ref = orc.pad_scale(case.x[idx].double().numpy(), case.meta["fft_size"], case.meta["scale"])
    want = torch.from_numpy(ref.astype(np.float32))
    assert torch.equal(_bits(y[torch.from_numpy(idx).cuda()].cpu()), _bits(want))


def run_moe(rw, dtype, tokens, experts, ld=None, off=0, seed=0, masked=False):
    ld = ld or experts
    g = np.random.default_rng(seed)
    # coarse values: ties, tied maxima included, are frequent
    s = np.round(g.standard_normal((tokens, ld)) * 3) / 4
    if masked:
        s[g.random((tokens, ld)) < 0.5] = -np.inf
        s[::7, :32] = -np.inf  # whole groups masked
    s_t = torch.from_numpy(s).to(dtype)
    es = ESIZE[dtype]
    G = 64
    sbuf = canary_tensor(G + off + tokens * ld + G, dtype)
    sbuf[G + off:G + off + tokens * ld] = s_t.reshape(-1).cuda()
    out = torch.full((tokens, experts // 32), float("nan"), dtype=torch.float32, device="cuda")
    st = rw.rowop_moe_group_top2(sbuf.data_ptr() + (G + off) * es, out.data_ptr(), tokens,
                                 experts, ld, rw.dtype_code(dtype),
                                 torch.cuda.current_stream().cuda_stream)
    assert st == 0, rw.STATUS.get(st, st)
    torch.cuda.synchronize()
    ref = orc.moe_group_top2(s_t[:, :experts].double().numpy())
    return out.cpu(), torch.from_numpy(ref.astype(np.float32))


MOE_CASES = [(1000, 256, None, 0, False), (333, 32, None, 0, False),
             (257, 288, None, 0, True), (100, 64, 72, 0, False),
             (97, 256, None, 1, True), (50000, 64, None, 0, False)]


@pytest.mark.parametrize("dtype", DTYPES, ids=DTYPE_IDS)
@pytest.mark.parametrize("case", MOE_CASES, ids=lambda c: f"{c[0]}x{c[1]}-ld{c[2]}-off{c[3]}")
def test_moe_group_top2_parity(rw, dtype, case):
    tokens, experts, ld, off, masked = case
    got, want = run_moe(rw, dtype, tokens, experts, ld, off, seed=tokens, masked=masked)
    assert torch.equal(_bits(got), _bits(want))


def test_moe_group_top2_ties(rw):
    """A tied maximum counts twice: the score is 2*max, not max + the next
    distinct value."""
    s = torch.zeros(4, 64)
    s[0, :32] = 1.0                 # all tied
    s[1, 3] = 5.0
    s[1, 17] = 5.0                  # tied maximum
    s[1, 20] = 4.0
    s[2, 40] = 7.0                  # unique maximum in group 1
    s[2, 41] = 6.0
    s[3, :] = -float("inf")
    s[3, 9] = 2.0                   # a single unmasked expert
    out = rw.moe_group_top2(s.cuda()).cpu()
    assert out[0, 0] == 2.0 and out[1, 0] == 10.0 and out[2, 1] == 13.0
    assert out[3, 0] == -float("inf") and out[3, 1] == -float("inf")


def test_moe_group_top2_workload_sampled(rw):
    from paper_2607_23089_gb300 import workloads as wl
    case = wl.moe_group()
    out = rw.moe_group_top2(case.x.cuda()).cpu()
    idx = np.random.default_rng(2).choice(case.x.shape[0], 2000, replace=False)
    ref = orc.moe_group_top2(case.x[idx].double().numpy())
    assert torch.equal(_bits(out[idx]), _bits(torch.from_numpy(ref.astype(np.float32))))
