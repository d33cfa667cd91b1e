"""Seeded synthetic inputs for the row-op workloads.

This module only draws random numbers; it holds none of the operators'
arithmetic, and both the CUDA path's tests/benchmark and the CPU oracle take
their inputs from it.  Every draw uses ``torch.Generator('cpu')`` seeded per
workload, in float32, in a fixed order: row lengths (ragged) -> x -> outlier
mask / sign -> per-row scale -> gamma -> beta.  bf16 tensors are made from the
float32 draws by round-to-nearest-even (``.to(torch.bfloat16)``).

The five workloads (rows x cols, dtype, distribution, seed):

1. ``softmax_1k``    fp32 softmax, 1024 x 1000, x = 4*N(0,1), seed 0.
2. ``short_rows``    fp32 softmax and log-softmax, 32768 x C for C in
   {64, 128, 256, 512}, x = 4*N(0,1), seed 1 (one generator per C).
3. ``medium_norm``   bf16 RMSNorm (eps 1e-6) and LayerNorm (eps 1e-5),
   8192 x 4096, x = N(0,1) * U(0.1, 10) per row, gamma = 1 + 0.1*N(0,1),
   beta = 0.1*N(0,1) per column, seed 2.
4. ``long_rows``     fp32 log-softmax, 256 x 262144, x = N(0,1) with each
   entry independently (p = 0.001) replaced by +80 or -80 (p = 1/2 each),
   seed 3.
5. ``ragged_ln``     bf16 LayerNorm (eps 1e-5) over 16384 ragged rows with
   lengths uniform on {1..32768} as int64 CSR offsets into one packed buffer,
   x = N(0,1) * U(0.1, 10) per row, gamma/beta of length 32768 drawn as in
   workload 3, seed 4.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Optional

import torch

ESIZE = {torch.float32: 4, torch.bfloat16: 2, torch.float16: 2}


@dataclass
class Case:
    """One operator call on one synthetic input (host tensors)."""
    name: str
    op: str                      # softmax | logsoftmax | layernorm | rmsnorm
    x: torch.Tensor              # dense: rows x cols; ragged: packed 1-D
    dtype: torch.dtype
    offsets: Optional[torch.Tensor] = None   # int64 [rows+1] when ragged
    gamma: Optional[torch.Tensor] = None
    beta: Optional[torch.Tensor] = None
    eps: float = 0.0
    max_len: int = 0
    meta: dict = field(default_factory=dict)
    resid: Optional[torch.Tensor] = None     # fused residual add: the residual r
    dy: Optional[torch.Tensor] = None        # backward passes: the upstream gradient

    @property
    def ragged(self) -> bool:
        return self.offsets is not None

    @property
    def rows(self) -> int:
        return (self.offsets.numel() - 1) if self.ragged else self.x.shape[0]

    @property
    def elements(self) -> int:
        return int(self.offsets[-1]) if self.ragged else self.x.numel()

    def algorithmic_bytes(self) -> int:
        """Bytes the operator must move: read x once, write y once, read
        gamma/beta once, read the offsets once."""
        es = ESIZE[self.dtype]
        if self.op.endswith("_backward"):
            # read the forward input (norms) or output (softmax family) and dy,
            # write dx; norms also read gamma and write dgamma (and dbeta)
            b = 3 * self.elements * es
            ncol = self.max_len if self.ragged else self.x.shape[1]
            if self.ragged:
                b += self.offsets.numel() * 8
            if self.op == "layernorm_backward":
                b += 3 * ncol * es
            elif self.op == "rmsnorm_backward":
                b += 2 * ncol * es
            return b
        if self.op == "pad_scale":  # read rows x seqlen, write rows x fft_size
            return self.x.numel() * es + self.x.shape[0] * self.meta["fft_size"] * es
        if self.op == "moe_group_top2":  # read the scores, write one float per group
            return self.x.numel() * es + self.x.shape[0] * (self.x.shape[1] // 32) * 4
        b = 2 * self.elements * es
        if self.resid is not None:  # also read r and write the sum
            b += 2 * self.elements * es
        ncol = self.max_len if self.ragged else self.x.shape[1]
        if self.gamma is not None:
            b += ncol * es
        if self.beta is not None:
            b += ncol * es
        if self.ragged:
            b += self.offsets.numel() * 8
        return b


def _gen(seed: int) -> torch.Generator:
    return torch.Generator("cpu").manual_seed(seed)


def _affine(g: torch.Generator, n: int, dtype):
    gamma = (1.0 + 0.1 * torch.randn(n, generator=g)).to(dtype)
    beta = (0.1 * torch.randn(n, generator=g)).to(dtype)
    return gamma, beta


def softmax_1k(rows: int = 1024, cols: int = 1000) -> Case:
    g = _gen(0)
    x = 4.0 * torch.randn(rows, cols, generator=g)
    return Case("softmax_1k", "softmax", x, torch.float32)


def short_rows(cols: int, op: str = "softmax", rows: int = 32768) -> Case:
    g = _gen(1)
    x = 4.0 * torch.randn(rows, cols, generator=g)
    return Case(f"short_rows_{op}_{cols}", op, x, torch.float32,
                meta={"cols": cols})


def medium_norm(op: str, rows: int = 8192, cols: int = 4096) -> Case:
    g = _gen(2)
    x = torch.randn(rows, cols, generator=g)
    scale = 0.1 + 9.9 * torch.rand(rows, 1, generator=g)
    x = (x * scale).to(torch.bfloat16)
    gamma, beta = _affine(g, cols, torch.bfloat16)
    if op == "rmsnorm":
        return Case(f"medium_norm_{op}", op, x, torch.bfloat16, gamma=gamma,
                    eps=1e-6)
    return Case(f"medium_norm_{op}", op, x, torch.bfloat16, gamma=gamma,
                beta=beta, eps=1e-5)


def long_rows(rows: int = 256, cols: int = 262144, op: str = "logsoftmax",
              p_outlier: float = 0.001, outlier: float = 80.0) -> Case:
    g = _gen(3)
    x = torch.randn(rows, cols, generator=g)
    mask = torch.rand(rows, cols, generator=g) < p_outlier
    sign = torch.rand(rows, cols, generator=g) < 0.5
    spike = torch.where(sign, torch.tensor(outlier), torch.tensor(-outlier))
    x = torch.where(mask, spike, x)
    return Case(f"long_rows_{op}", op, x, torch.float32)


def ragged_lengths(rows: int, max_len: int, g: torch.Generator,
                   min_len: int = 1) -> torch.Tensor:
    return torch.randint(min_len, max_len + 1, (rows,), generator=g,
                         dtype=torch.int64)


def offsets_from_lengths(lengths: torch.Tensor) -> torch.Tensor:
    off = torch.zeros(lengths.numel() + 1, dtype=torch.int64)
    off[1:] = torch.cumsum(lengths, 0)
    return off


def ragged_ln(rows: int = 16384, max_len: int = 32768, op: str = "layernorm",
              dtype=torch.bfloat16, seed: int = 4) -> Case:
    g = _gen(seed)
    lengths = ragged_lengths(rows, max_len, g)
    off = offsets_from_lengths(lengths)
    total = int(off[-1])
    x = torch.randn(total, generator=g)
    scale = 0.1 + 9.9 * torch.rand(rows, generator=g)
    x = (x * torch.repeat_interleave(scale, lengths)).to(dtype)
    gamma, beta = _affine(g, max_len, dtype)
    eps = {"layernorm": 1e-5, "rmsnorm": 1e-6}.get(op, 0.0)
    return Case(f"ragged_{op}", op, x, dtype, offsets=off,
                gamma=gamma if op in ("layernorm", "rmsnorm") else None,
                beta=beta if op == "layernorm" else None,
                eps=eps, max_len=max_len)


def medium_add_norm(op: str, rows: int = 8192, cols: int = 4096, seed: int = 7) -> Case:
    """Fused residual add + norm on the workload-3 shape: bf16 x as in
    workload 3, residual r = N(0,1), gamma/beta as there.  Not one of the five
    workloads."""
    g = _gen(seed)
    x = torch.randn(rows, cols, generator=g)
    scale = 0.1 + 9.9 * torch.rand(rows, 1, generator=g)
    x = (x * scale).to(torch.bfloat16)
    r = torch.randn(rows, cols, generator=g).to(torch.bfloat16)
    gamma, beta = _affine(g, cols, torch.bfloat16)
    if op == "rmsnorm":
        return Case("medium_add_rmsnorm", "add_rmsnorm", x, torch.bfloat16, gamma=gamma,
                    eps=1e-6, resid=r)
    return Case("medium_add_layernorm", "add_layernorm", x, torch.bfloat16, gamma=gamma,
                beta=beta, eps=1e-5, resid=r)


def hyena_pad(rows: int = 16384, seqlen: int = 4096, fft_size: int = 8192,
              seed: int = 5) -> Case:
    """Hyena FFT-size padding (§6): fp32 rows x seqlen, x = N(0,1), padded
    with zeros to fft_size = 2*seqlen and scaled by 1/fft_size (the usual
    normalisation of an FFT convolution).  Not one of the five workloads
    above; the shapes are those of a long-convolution layer (rows = batch x
    channels)."""
    g = _gen(seed)
    x = torch.randn(rows, seqlen, generator=g)
    return Case("hyena_pad_scale", "pad_scale", x, torch.float32,
                meta={"fft_size": fft_size, "scale": 1.0 / fft_size})


def moe_group(tokens: int = 131072, experts: int = 256, seed: int = 6,
              dtype=torch.float32) -> Case:
    """MoE group score (§2.1): tokens x 256 expert scores in 8 groups of 32,
    s = sigmoid(N(0,1)) rounded to multiples of 1/256 so that ties, tied
    maxima included, are common.  Not one of the five workloads above."""
    g = _gen(seed)
    s = torch.sigmoid(torch.randn(tokens, experts, generator=g))
    s = torch.round(s * 256) / 256
    return Case("moe_group_top2", "moe_group_top2", s.to(dtype), dtype)


def norm_backward(op: str, rows: int = 8192, cols: int = 4096, seed: int = 8) -> Case:
    """Backward of a workload-3 norm: bf16 x drawn as in workload 3, upstream
    gradient dy = N(0,1), gamma as there; the gradients are dx, dgamma (and
    dbeta for LayerNorm).  Not one of the five workloads."""
    g = _gen(seed)
    x = torch.randn(rows, cols, generator=g)
    scale = 0.1 + 9.9 * torch.rand(rows, 1, generator=g)
    x = (x * scale).to(torch.bfloat16)
    dy = torch.randn(rows, cols, generator=g).to(torch.bfloat16)
    gamma, _ = _affine(g, cols, torch.bfloat16)
    return Case(f"medium_norm_backward_{op}", f"{op}_backward", x, torch.bfloat16, gamma=gamma,
                eps=1e-5 if op == "layernorm" else 1e-6, dy=dy)


def softmax_backward(op: str = "softmax", rows: int = 32768, cols: int = 1024,
                     seed: int = 9) -> Case:
    """Backward of softmax / log-softmax over fp32 rows of 1024 (attention-row
    length): x = 4*N(0,1) is the FORWARD input -- the backward takes the
    forward output y = op(x), which the caller forms -- and dy = N(0,1).  Not
    one of the five workloads."""
    g = _gen(seed)
    x = 4.0 * torch.randn(rows, cols, generator=g)
    dy = torch.randn(rows, cols, generator=g)
    return Case(f"{op}_backward_{cols}", f"{op}_backward", x, torch.float32, dy=dy)


def ragged_softmax_backward(rows: int = 32768, max_len: int = 4096, seed: int = 10) -> Case:
    """Softmax backward over ragged fp32 rows (variable-length attention rows):
    lengths uniform on {1..max_len} as int64 CSR offsets, x = 4*N(0,1) the
    forward input (y = softmax(x) is formed by the caller), dy = N(0,1).  Not
    one of the five workloads."""
    g = _gen(seed)
    lengths = ragged_lengths(rows, max_len, g)
    off = offsets_from_lengths(lengths)
    total = int(off[-1])
    x = 4.0 * torch.randn(total, generator=g)
    dy = torch.randn(total, generator=g)
    return Case("ragged_softmax_backward", "softmax_backward", x, torch.float32, offsets=off,
                max_len=max_len, dy=dy)


def ragged_norm_backward(op: str = "layernorm", rows: int = 16384, max_len: int = 32768,
                         seed: int = 11) -> Case:
    """Backward of a norm over the ragged rows of workload 5: bf16 x drawn as
    there (lengths uniform on {1..max_len}, a scale per row), dy = N(0,1),
    gamma of max_len; the gradients are dx, dgamma (and dbeta for LayerNorm)
    of max_len columns.  Not one of the five workloads."""
    g = _gen(seed)
    lengths = ragged_lengths(rows, max_len, g)
    off = offsets_from_lengths(lengths)
    total = int(off[-1])
    x = torch.randn(total, generator=g)
    scale = 0.1 + 9.9 * torch.rand(rows, generator=g)
    x = (x * torch.repeat_interleave(scale, lengths)).to(torch.bfloat16)
    dy = torch.randn(total, generator=g).to(torch.bfloat16)
    gamma, _ = _affine(g, max_len, torch.bfloat16)
    return Case(f"ragged_{op}_backward", f"{op}_backward", x, torch.bfloat16, offsets=off,
                gamma=gamma, eps=1e-5 if op == "layernorm" else 1e-6, max_len=max_len, dy=dy)


def all_cases(scale_down: int = 1):
    """The five workloads as a flat list of cases.  ``scale_down`` > 1 divides
    every row count (not the row lengths) for quicker runs."""
    s = max(1, int(scale_down))
    out = [softmax_1k(rows=max(1, 1024 // s))]
    for c in (64, 128, 256, 512):
        for op in ("softmax", "logsoftmax"):
            out.append(short_rows(c, op, rows=max(1, 32768 // s)))
    for op in ("rmsnorm", "layernorm"):
        out.append(medium_norm(op, rows=max(1, 8192 // s)))
    out.append(long_rows(rows=max(1, 256 // s)))
    out.append(ragged_ln(rows=max(1, 16384 // s)))
    for op in ("rmsnorm", "layernorm"):
        out.append(medium_add_norm(op, rows=max(1, 8192 // s)))
    out.append(hyena_pad(rows=max(1, 16384 // s)))
    out.append(moe_group(tokens=max(1, 131072 // s)))
    for op in ("layernorm", "rmsnorm"):
        out.append(norm_backward(op, rows=max(1, 8192 // s)))
    for op in ("softmax", "logsoftmax"):
        out.append(softmax_backward(op, rows=max(1, 32768 // s)))
    out.append(ragged_softmax_backward(rows=max(1, 32768 // s)))
    for op in ("layernorm", "rmsnorm"):
        out.append(ragged_norm_backward(op, rows=max(1, 16384 // s)))
    return out


def by_name(name: str) -> Case:
    """Builds one workload case from its name (as in all_cases())."""
    if name.startswith("medium_norm_backward_"):
        return norm_backward(name[len("medium_norm_backward_"):])
    if name == "ragged_softmax_backward":
        return ragged_softmax_backward()
    if name in ("ragged_layernorm_backward", "ragged_rmsnorm_backward"):
        return ragged_norm_backward(name.split("_")[1])
    if name.startswith(("softmax_backward_", "logsoftmax_backward_")):
        op, _, cols = name.split("_")
        return softmax_backward(op, cols=int(cols))
    if name == "softmax_1k":
        return softmax_1k()
    if name.startswith("short_rows_"):
        _, _, op, cols = name.split("_")
        return short_rows(int(cols), op)
    if name.startswith("medium_norm_"):
        return medium_norm(name[len("medium_norm_"):])
    if name.startswith("long_rows_"):
        return long_rows(op=name[len("long_rows_"):])
    if name.startswith("ragged_"):
        return ragged_ln(op=name[len("ragged_"):])
    if name.startswith("medium_add_"):
        return medium_add_norm(name[len("medium_add_"):])
    if name == "hyena_pad_scale":
        return hyena_pad()
    if name == "moe_group_top2":
        return moe_group()
    raise KeyError(name)
