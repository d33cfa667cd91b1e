"""Plant plausible mistakes in a copy of the oracle (on the CPU) and check
that the pin suite catches every one.  The real oracle is never modified:
each mutant is compiled from an edited copy of the C source in a temporary
directory and loaded through a fresh copy of the Python wrapper."""
import importlib.util
import os
import re

import pytest

from tests.oracle_pins import ALL_PINS

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "rowop_oracle.c")
SRC_PM = os.path.join(ROOT, "oracle", "pad_moe_oracle.c")
SRC_BW = os.path.join(ROOT, "oracle", "backward_oracle.c")
WRAPPER = os.path.join(ROOT, "oracle", "rowop_oracle.py")

# (function whose body is edited, text, replacement, what the mistake is)
MUTANTS = [
    ("softmax_row", "s += exp(x[j] - m);", "s += exp(x[j]);",
     "sum without the max shift"),
    ("softmax_row", "y[j] = exp(x[j] - m) / s;", "y[j] = exp(x[j] - m) * s;",
     "multiply instead of divide"),
    ("softmax_row", "if (x[j] > m)", "if (x[j] < m)", "min instead of max"),
    ("logsoftmax_row", "(x[j] - m) - log_s", "(x[j] - m) + log_s",
     "wrong sign of log-sum"),
    ("logsoftmax_row", "(x[j] - m) - log_s", "x[j] - log_s",
     "dropped max term"),
    ("layernorm_row", "sq / (double)n", "sq / (double)(n - 1)",
     "unbiased variance"),
    ("layernorm_row", "sqrt(var + eps)", "(sqrt(var) + eps)",
     "eps outside the root"),
    ("layernorm_row", "* gamma[j] + beta[j]", "* gamma[j]", "dropped beta"),
    ("layernorm_row", "gamma[j]", "gamma[0]", "gamma index"),
    ("layernorm_row", "(x[j] - mu) / den", "(x[j] - mu) * den",
     "inverted scale"),
    ("rmsnorm_row", "sq / (double)n", "sq", "sum instead of mean of squares"),
    ("rmsnorm_row", "sqrt(ms + eps)", "sqrt(ms)", "dropped eps"),
    ("rmsnorm_row", "* gamma[j]", "", "dropped gamma"),
    ("oracle_softmax_ragged", "off[r + 1] - off[r]", "off[r + 1] - off[r] - 1",
     "ragged row length off by one"),
    ("oracle_layernorm_ragged", "gamma, beta,", "gamma + off[r], beta,",
     "gamma indexed by packed offset"),
    ("oracle_bucket", "bytes <= 4096", "bytes < 4096",
     "SMALL threshold off by one"),
    ("oracle_bucket", "bytes <= 32768", "bytes <= 65536",
     "MEDIUM threshold"),
    ("oracle_pad_scale", "c < seqlen ?", "c <= seqlen - 2 ?", "last live column zeroed"),
    ("oracle_pad_scale", "scale * x[r * seqlen + c]", "x[r * seqlen + c]", "scale dropped"),
    ("oracle_pad_scale", "x[r * seqlen + c]", "x[r * seqlen + (seqlen - 1 - c)]",
     "row read backwards"),
    ("oracle_moe_group_top2", "if (i != j && ", "if (", "pair of a score with itself"),
    ("oracle_moe_group_top2", "g * group", "g", "groups overlap"),
    ("oracle_moe_group_top2", "j < group;", "j < group - 1 && i < group - 1;",
     "last member skipped"),
    ("oracle_moe_group_top2", "w[i] + w[j] > best", "w[i] + w[j] >= best + 1.0",
     "comparison off"),
    ("softmax_bwd_row", "(dy[j] - s)", "(dy[j] + s)", "softmax backward sign"),
    ("softmax_bwd_row", "s += dy[j] * y[j];", "s += dy[j];", "softmax backward dot without y"),
    ("logsoftmax_bwd_row", "exp(y[j]) * s", "y[j] * s", "log-softmax backward without exp"),
    ("layernorm_bwd_row", "- a - xhat * b", "- xhat * b", "LayerNorm backward mean term dropped"),
    ("layernorm_bwd_row", "rstd * (dy[j]", "(dy[j]", "LayerNorm backward rstd factor dropped"),
    ("layernorm_bwd_row", "sgx += g * ((x[j] - mu) * rstd);", "sgx += g * (x[j] - mu);",
     "LayerNorm backward xhat without rstd"),
    ("layernorm_bwd_row", "dy[j] * gamma[j] - a", "dy[j] - a", "LayerNorm backward gamma dropped"),
    ("layernorm_stats", "sq / (double)n + eps", "sq / (double)(n - 1) + eps",
     "LayerNorm backward unbiased variance"),
    ("oracle_layernorm_backward", "sg += dy[r * cols + j] * xhat;", "sg += dy[r * cols + j];",
     "dgamma without xhat"),
    ("oracle_layernorm_backward", "for (int64_t r = 0; r < rows; ++r) {\n            const",
     "for (int64_t r = 1; r < rows; ++r) {\n            const", "column sums skip row 0"),
    ("rmsnorm_bwd_row", "- (x[j] * rstd) * b", "- x[j] * b", "RMSNorm backward xhat without rstd"),
    ("rmsnorm_rstd", "sq / (double)n + eps", "sq + eps", "RMSNorm backward sum of squares"),
    ("oracle_rmsnorm_backward", "(x[r * cols + j] * rs[r])", "x[r * cols + j]",
     "RMSNorm dgamma uses x"),
]

# functions defined in pad_moe_oracle.c rather than rowop_oracle.c
PM_FUNCS = {"oracle_pad_scale", "oracle_moe_group_top2"}
# functions defined in backward_oracle.c
BW_FUNCS = {"softmax_bwd_row", "logsoftmax_bwd_row", "layernorm_bwd_row", "layernorm_stats",
            "oracle_layernorm_backward", "rmsnorm_bwd_row", "rmsnorm_rstd",
            "oracle_rmsnorm_backward"}


def _mutate(src: str, func: str, old: str, new: str) -> str:
    m = re.search(r"\n[a-z ]*\b" + re.escape(func) + r"\(", src)
    assert m, func
    start = m.start()
    end = src.index("\n}\n", start)
    body = src[start:end]
    assert old in body, (func, old)
    return src[:start] + body.replace(old, new, 1) + src[end:]


def _load_mutant(tmp_path, text, text_pm, text_bw):
    d = tmp_path / "mut"
    d.mkdir()
    (d / "rowop_oracle.c").write_text(text)
    (d / "pad_moe_oracle.c").write_text(text_pm)
    (d / "backward_oracle.c").write_text(text_bw)
    spec = importlib.util.spec_from_file_location("oracle_mutant", WRAPPER)
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    mod._SRC = str(d / "rowop_oracle.c")
    mod._SRCS = [str(d / "rowop_oracle.c"), str(d / "pad_moe_oracle.c"),
                 str(d / "backward_oracle.c")]
    mod._BUILD_DIR = str(d / "_build")
    mod._LIB_PATH = str(d / "_build" / "liboracle.so")
    mod._lib = None
    return mod


@pytest.mark.parametrize("func,old,new,what", MUTANTS,
                         ids=[m[3].replace(" ", "_") for m in MUTANTS])
def test_pins_catch_mutant(tmp_path, func, old, new, what):
    with open(SRC) as f:
        src = f.read()
    with open(SRC_PM) as f:
        src_pm = f.read()
    with open(SRC_BW) as f:
        src_bw = f.read()
    if func in PM_FUNCS:
        src_pm = _mutate(src_pm, func, old, new)
    elif func in BW_FUNCS:
        src_bw = _mutate(src_bw, func, old, new)
    else:
        src = _mutate(src, func, old, new)
    mod = _load_mutant(tmp_path, src, src_pm, src_bw)
    caught = []
    for pin in ALL_PINS:
        try:
            pin(mod)
        except (AssertionError, ValueError, FloatingPointError) as e:
            caught.append(pin.__name__)
    assert caught, f"no pin caught the planted mistake: {what}"


# Mistakes planted in the Python composition of the ragged norm backward
# (rowop_oracle.py, _ragged_norm_backward): (text, replacement, what).
RAGGED_BWD_MUTANTS = [
    ("g[:b - a]", "g[1:b - a + 1]", "gamma taken one column late"),
    ("s[:b - a] += part", "s[-(b - a):] += part", "column sums aligned to the row end"),
    ("range(off.shape[0] - 1)", "range(off.shape[0] - 2)", "last row left out"),
    ("zip(sums, out[1:])", "zip(sums, out[1:2])", "dbeta never summed"),
    ("dx[a:b] = out[0][0]", "dx[a:b] = out[0][0][::-1]", "dx of a row reversed"),
    ("if b == a:\n            continue", "if b - a < 2:\n            continue",
     "one-element rows skipped"),
]


@pytest.mark.parametrize("old,new,what", RAGGED_BWD_MUTANTS,
                         ids=[m[2].replace(" ", "_") for m in RAGGED_BWD_MUTANTS])
def test_pins_catch_ragged_backward_mutant(tmp_path, old, new, what):
    """The composition is Python, so the mutant is an edited copy of the
    wrapper that loads the real (unmodified) compiled oracle."""
    from oracle import rowop_oracle as real
    real.build()
    with open(WRAPPER) as f:
        text = f.read()
    start = text.index("def _ragged_norm_backward(")
    end = text.index("\ndef ", start + 1)
    body = text[start:end]
    assert old in body, old
    path = tmp_path / "oracle_ragged_mutant.py"
    path.write_text(text[:start] + body.replace(old, new, 1) + text[end:])
    spec = importlib.util.spec_from_file_location("oracle_ragged_mutant", str(path))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    mod._SRCS = real._SRCS
    mod._BUILD_DIR = real._BUILD_DIR
    mod._LIB_PATH = real._LIB_PATH
    mod._lib = None
    caught = []
    for pin in ALL_PINS:
        try:
            pin(mod)
        except (AssertionError, ValueError, FloatingPointError):
            caught.append(pin.__name__)
    assert caught, f"no pin caught the planted mistake: {what}"
