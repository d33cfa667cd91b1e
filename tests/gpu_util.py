"""Helpers for the GPU parity tests: guarded device buffers, oracle calls and
the tolerance check.

Tolerances (per element, against the double-precision oracle):
  fp32   |gpu - ref| <= 1e-6 + 1e-5 * |ref|
  bf16   |gpu - ref| <= 1e-6 + 1e-2 * |ref|   (bf16 I/O, fp32 arithmetic)
NaN must appear exactly where the oracle has NaN.
"""
from __future__ import annotations

import numpy as np
import torch

from oracle import rowop_oracle as orc

TOL = {torch.float32: (1e-5, 1e-6), torch.bfloat16: (1e-2, 1e-6),
       torch.float16: (1e-3, 1e-6)}
CANARY = {torch.float32: 0x7FC0DEAD, torch.bfloat16: 0x7FC1, torch.float16: 0x7FC1}
ESIZE = {torch.float32: 4, torch.bfloat16: 2, torch.float16: 2}
NORM_OPS = ("layernorm", "rmsnorm")
ALL_OPS = ("softmax", "logsoftmax", "layernorm", "rmsnorm")
DTYPES = (torch.float32, torch.bfloat16, torch.float16)
DTYPE_IDS = ["f32", "bf16", "f16"]


def assert_close(got, ref, dtype, what=""):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, (got.shape, ref.shape)
    rtol, atol = TOL[dtype]
    nan_g, nan_r = np.isnan(got), np.isnan(ref)
    assert (nan_g == nan_r).all(), f"{what}: NaN pattern differs"
    inf_g, inf_r = np.isinf(got), np.isinf(ref)
    assert (inf_g == inf_r).all(), f"{what}: infinity pattern differs"
    assert (got[inf_r] == ref[inf_r]).all(), f"{what}: infinity of the wrong sign"
    special = nan_r | inf_r
    err = np.abs(np.where(special, 0.0, got - np.where(special, 0.0, ref)))
    lim = atol + rtol * np.abs(np.where(special, 0.0, ref))
    bad = err > lim
    if bad.any():
        i = np.unravel_index(np.argmax(err - lim), err.shape)
        raise AssertionError(
            f"{what}: {int(bad.sum())} of {bad.size} elements out of tolerance; "
            f"worst at {i}: got {got[i]!r} ref {ref[i]!r} err {err[i]:.3e} "
            f"lim {lim[i]:.3e}")


def canary_tensor(n, dtype, device="cuda"):
    """A device buffer of n elements filled with a NaN bit pattern."""
    if dtype == torch.float32:
        raw = torch.full((n,), CANARY[dtype], dtype=torch.int32, device=device)
        return raw.view(torch.float32)
    raw = torch.full((n,), CANARY[dtype], dtype=torch.int16, device=device)
    return raw.view(dtype)


def is_canary(t):
    dtype = t.dtype
    if dtype == torch.float32:
        return t.view(torch.int32) == CANARY[dtype]
    return t.view(torch.int16) == CANARY[dtype]


def to_f64(t):
    return t.detach().to("cpu").double().numpy()


def oracle_dense(op, x64, g64=None, b64=None, eps=0.0):
    if op == "softmax":
        return orc.softmax(x64)
    if op == "logsoftmax":
        return orc.logsoftmax(x64)
    if op == "layernorm":
        return orc.layernorm(x64, g64, b64, eps=eps)
    return orc.rmsnorm(x64, g64, eps=eps)


def oracle_ragged(op, x64, off, g64=None, b64=None, eps=0.0):
    if op == "softmax":
        return orc.softmax_ragged(x64, off)
    if op == "logsoftmax":
        return orc.logsoftmax_ragged(x64, off)
    if op == "layernorm":
        return orc.layernorm_ragged(x64, off, g64, b64, eps=eps)
    return orc.rmsnorm_ragged(x64, off, g64, eps=eps)


def eps_for(op):
    return {"layernorm": 1e-5, "rmsnorm": 1e-6}.get(op, 0.0)


def gen(shape, dtype, seed, scale=3.0):
    g = torch.Generator("cpu").manual_seed(seed)
    return (scale * torch.randn(*shape, generator=g)).to(dtype)


def gen_affine(n, dtype, seed):
    g = torch.Generator("cpu").manual_seed(seed + 7919)
    gamma = (1.0 + 0.1 * torch.randn(n, generator=g)).to(dtype)
    beta = (0.1 * torch.randn(n, generator=g)).to(dtype)
    return gamma, beta
