"""The five synthetic workloads at full size, called exactly as the benchmark
calls them, checked against the oracle (every element for workloads 1-3,
every 8th row for 4, every 16th row for the ragged workload 5), plus the
status path of the bounded device waits."""
import numpy as np
import pytest
import torch

from paper_2607_23089_gb300 import workloads as wl
from tests.gpu_util import assert_close, oracle_dense, oracle_ragged, to_f64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def rw():
    from paper_2607_23089_gb300 import build, rowop
    build.build()
    rowop.load()
    torch.cuda.set_device(0)
    return rowop


def _dense(rw, case, row_step=1):
    x = case.x.cuda()
    g = case.gamma.cuda() if case.gamma is not None else None
    b = case.beta.cuda() if case.beta is not None else None
    y = rw.run(case.op, x, gamma=g, beta=b, eps=case.eps)
    assert rw.check_status() == 0
    sel = slice(None, None, row_step)
    ref = oracle_dense(case.op, case.x[sel].double().numpy(),
                       None if g is None else case.gamma.double().numpy(),
                       None if b is None else case.beta.double().numpy(), case.eps)
    assert_close(to_f64(y[sel]), ref, case.dtype, case.name)


def test_workload_softmax_1k(rw):
    _dense(rw, wl.softmax_1k())


@pytest.mark.parametrize("cols", [64, 128, 256, 512])
@pytest.mark.parametrize("op", ["softmax", "logsoftmax"])
def test_workload_short_rows(rw, op, cols):
    _dense(rw, wl.short_rows(cols, op))


@pytest.mark.parametrize("op", ["rmsnorm", "layernorm"])
def test_workload_medium_norm(rw, op):
    _dense(rw, wl.medium_norm(op))


def test_workload_long_rows(rw):
    _dense(rw, wl.long_rows(), row_step=8)


def test_workload_ragged_ln(rw):
    case = wl.ragged_ln()
    x = case.x.cuda()
    off = case.offsets.cuda()
    y = rw.layernorm_ragged(x, off, case.max_len, case.gamma.cuda(), case.beta.cuda(),
                            case.eps)
    assert rw.check_status() == 0
    offs = case.offsets.numpy()
    pick = np.arange(0, case.rows, 16)
    lens = offs[pick + 1] - offs[pick]
    sub_off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    xs = np.concatenate([case.x[offs[i]:offs[i + 1]].double().numpy() for i in pick])
    ys = np.concatenate([to_f64(y[offs[i]:offs[i + 1]]) for i in pick])
    ref = oracle_ragged("layernorm", xs, sub_off, case.gamma.double().numpy(),
                        case.beta.double().numpy(), case.eps)
    assert_close(ys, ref, case.dtype, "ragged_ln (every 16th row)")


def test_bounded_wait_reports_timeout(rw):
    """A wait that nothing completes runs out after its limit, the kernel
    returns, the status reads ROWOP_ERR_TIMEOUT once, and the context stays
    usable."""
    assert rw.check_status() == 0
    s = torch.cuda.current_stream().cuda_stream
    assert rw.rowop_debug_wait_timeout(20_000_000, s) == 0  # 20 ms
    assert rw.check_status() == rw.ROWOP_ERR_TIMEOUT
    assert rw.check_status() == 0
    x = torch.randn(8, 100, device="cuda")
    torch.testing.assert_close(rw.softmax(x), torch.softmax(x, 1), rtol=1e-5, atol=1e-6)
