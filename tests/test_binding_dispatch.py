"""rowop.run() sends each operator to the helper for its layout (dense, or
ragged when offsets are given), checked on the CPU with the helpers replaced
by recorders (nothing reaches the library)."""
import pytest

from paper_2607_23089_gb300 import rowop


@pytest.fixture
def calls(monkeypatch):
    seen = []

    def recorder(name, result):
        def fn(*args, **kwargs):
            seen.append((name, args, kwargs))
            return result
        return fn

    for name in ("softmax_backward", "logsoftmax_backward", "softmax_backward_ragged"):
        monkeypatch.setattr(rowop, name, recorder(name, "dx"))
    for name in ("layernorm_backward", "layernorm_backward_ragged"):
        monkeypatch.setattr(rowop, name, recorder(name, ("dx", "dg", "db")))
    for name in ("rmsnorm_backward", "rmsnorm_backward_ragged"):
        monkeypatch.setattr(rowop, name, recorder(name, ("dx", "dg")))
    return seen


@pytest.mark.parametrize("op,dense,ragged", [
    ("softmax_backward", "softmax_backward", "softmax_backward_ragged"),
    ("logsoftmax_backward", "logsoftmax_backward", "softmax_backward_ragged"),
    ("layernorm_backward", "layernorm_backward", "layernorm_backward_ragged"),
    ("rmsnorm_backward", "rmsnorm_backward", "rmsnorm_backward_ragged"),
])
def test_backward_ops_follow_the_layout(calls, op, dense, ragged):
    assert rowop.run(op, "x", dy="dy") == "dx"
    assert calls[-1][0] == dense
    assert rowop.run(op, "x", dy="dy", offsets="off", max_len=77, ws="ws") == "dx"
    name, args, kwargs = calls[-1]
    assert name == ragged
    assert args[:4] == ("x", "dy", "off", 77) and kwargs.get("ws") == "ws"
    if op.startswith("log"):
        assert kwargs.get("log") is True
    elif op == "softmax_backward":
        assert kwargs.get("log") is False


@pytest.mark.parametrize("op", ["pad_scale", "add_layernorm", "add_rmsnorm", "moe_group_top2"])
def test_dense_only_ops_refuse_offsets(op):
    with pytest.raises(ValueError, match="no ragged form"):
        rowop.run(op, "x", offsets="off", max_len=8)
