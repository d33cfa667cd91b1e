"""rowop_layernorm_ragged_static, the ragged LayerNorm entry point that takes
its workspace from a fixed array inside the library instead of caller
memory, for callers that cannot allocate one (a plugin that is handed only
its input and output buffers, a path that may not call cudaMalloc).  Called through the C ABI and compared, bit for bit, with
rowop_layernorm_ragged on a caller-owned workspace, on calls made one after
another (so any state left over from the previous call would show), at the
largest row count it accepts, and one row beyond it (rejected).  Collected
last so that it also runs after every other GPU test in the same process."""
import os
import re

import numpy as np
import pytest
import torch

from tests.gpu_util import assert_close, canary_tensor, gen_affine, oracle_ragged, to_f64

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def static_max_rows():
    text = open(os.path.join(ROOT, "include", "rowop.h")).read()
    return int(re.search(r"#define\s+ROWOP_STATIC_MAX_ROWS\s+(\d+)", text).group(1))


@pytest.fixture(scope="module")
def rw():
    from paper_2607_23089_gb300 import build, rowop
    build.build()
    rowop.load()
    torch.cuda.set_device(0)
    return rowop


def bits(t):
    return t.view(torch.int32 if t.dtype == torch.float32 else torch.int16).cpu()


def both_calls(rw, x, off, rows, max_len, gam, bet, dtype, eps):
    """Runs the caller-workspace call and the static-workspace call on the same
    inputs into separate canary-filled outputs; returns both outputs."""
    code = rw.dtype_code(dtype)
    s = torch.cuda.current_stream().cuda_stream
    y_ref = canary_tensor(x.numel(), dtype)
    y_st = canary_tensor(x.numel(), dtype)
    ws = rw.ragged_workspace(rows)
    gp = None if gam is None else gam.data_ptr()
    bp = None if bet is None else bet.data_ptr()
    st = rw.rowop_layernorm_ragged(x.data_ptr(), y_ref.data_ptr(), gp, bp, off.data_ptr(), rows,
                                   max_len, code, eps, ws.data_ptr(), ws.numel(), s)
    assert st == rw.ROWOP_OK, rw.rowop_status_string(st)
    st = rw.rowop_layernorm_ragged_static(x.data_ptr(), y_st.data_ptr(), gp, bp, off.data_ptr(),
                                          rows, max_len, code, eps, s)
    assert st == rw.ROWOP_OK, rw.rowop_status_string(st)
    assert rw.rowop_check_status(s) == rw.ROWOP_OK
    return y_ref, y_st


def test_static_workspace_equals_caller_workspace(rw):
    # call 1: bf16, every bucket (empty, SMALL, MEDIUM, cluster-split LARGE)
    g = np.random.default_rng(2024)
    max_len = 40000
    lens = g.integers(0, max_len + 1, size=700)
    lens[:40] = g.integers(0, 3, size=40)
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    total = int(off[-1])
    gx = torch.Generator("cpu").manual_seed(5)
    x = (3.0 * torch.randn(total, generator=gx) + 1.5).to(torch.bfloat16).cuda()
    gam, bet = gen_affine(max_len, torch.bfloat16, 5)
    gam, bet = gam.cuda(), bet.cuda()
    off_d = torch.from_numpy(off).cuda()
    y_ref, y_st = both_calls(rw, x, off_d, lens.size, max_len, gam, bet, torch.bfloat16, 1e-5)
    assert torch.equal(bits(y_ref), bits(y_st))
    ref = oracle_ragged("layernorm", to_f64(x), off, to_f64(gam), to_f64(bet), eps=1e-5)
    assert_close(to_f64(y_st), ref, torch.bfloat16, "static workspace, call 1")

    # call 2, right after: fp32, a different row count and a non-zero first
    # offset, no affine parameters
    lens2 = g.integers(1, 9000, size=1500)
    off2 = (37 + np.concatenate([[0], np.cumsum(lens2)])).astype(np.int64)
    x2 = torch.randn(int(off2[-1]) + 11, generator=gx).cuda()
    off2_d = torch.from_numpy(off2).cuda()
    y_ref2, y_st2 = both_calls(rw, x2, off2_d, lens2.size, 9000, None, None, torch.float32, 1e-5)
    assert torch.equal(bits(y_ref2), bits(y_st2))
    # the elements before the first row and after the last stay untouched
    assert torch.equal(bits(y_st2)[:37], bits(canary_tensor(37, torch.float32)))
    assert torch.equal(bits(y_st2)[-11:], bits(canary_tensor(11, torch.float32)))


def test_static_workspace_row_limit(rw):
    nmax = static_max_rows()
    s = torch.cuda.current_stream().cuda_stream
    # exactly the limit: accepted, equal to the caller-workspace call
    g = np.random.default_rng(7)
    lens = g.integers(0, 48, size=nmax)
    off = torch.from_numpy(np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)).cuda()
    x = torch.randn(int(lens.sum()), generator=torch.Generator("cpu").manual_seed(8)).cuda()
    gam, bet = gen_affine(48, torch.float32, 8)
    y_ref, y_st = both_calls(rw, x, off, nmax, 47, gam.cuda(), bet.cuda(), torch.float32, 1e-5)
    assert torch.equal(bits(y_ref), bits(y_st))
    # one row more: rejected before anything is launched (the offsets are all
    # zero, so even a launch would touch nothing)
    zeros = torch.zeros(nmax + 2, dtype=torch.int64, device="cuda")
    y = canary_tensor(16, torch.float32)
    st = rw.rowop_layernorm_ragged_static(y.data_ptr(), y.data_ptr(), None, None,
                                          zeros.data_ptr(), nmax + 1, 16,
                                          rw.ROWOP_F32, 1e-5, s)
    assert st == rw.ROWOP_ERR_WORKSPACE
    assert rw.rowop_check_status(s) == rw.ROWOP_OK
    # argument errors are the caller-workspace call's
    assert rw.rowop_layernorm_ragged_static(y.data_ptr(), y.data_ptr(), None, None,
                                            zeros.data_ptr(), -1, 16, rw.ROWOP_F32, 1e-5,
                                            s) == rw.ROWOP_ERR_INVALID_ARG
    assert rw.rowop_layernorm_ragged_static(y.data_ptr(), y.data_ptr(), None, None,
                                            zeros.data_ptr(), 0, 16, rw.ROWOP_F32, 1e-5,
                                            s) == rw.ROWOP_OK
