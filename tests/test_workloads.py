"""The synthetic input recipe, on the CPU: the headline ragged workload's
lengths (drawn first from its seed, as the generator does) give the stated
total and bucket counts, its algorithmic bytes are the benchmark's figure,
and the generators are pure functions of their seeds."""
import numpy as np
import torch

from oracle import rowop_oracle as orc
from paper_2607_23089_gb300 import workloads as wl


def test_headline_ragged_lengths_and_buckets():
    g = wl._gen(4)
    lengths = wl.ragged_lengths(16384, 32768, g).numpy()
    assert lengths.shape == (16384,)
    assert lengths.min() >= 1 and lengths.max() <= 32768
    assert int(lengths.sum()) == 270_408_470
    counts = np.bincount([orc.bucket(int(n), 2) for n in lengths], minlength=3)
    assert counts.tolist() == [1014, 7110, 8260]


def test_headline_algorithmic_bytes():
    g = wl._gen(4)
    off = wl.offsets_from_lengths(wl.ragged_lengths(16384, 32768, g))
    gamma = torch.zeros(32768, dtype=torch.bfloat16)
    case = wl.Case("ragged_layernorm", "layernorm", torch.empty(0, dtype=torch.bfloat16),
                   torch.bfloat16, offsets=off, gamma=gamma, beta=gamma, eps=1e-5,
                   max_len=32768)
    # read x and write y once (2 bytes each), gamma and beta once, the offsets once
    assert case.algorithmic_bytes() == 2 * 270_408_470 * 2 + 2 * 32768 * 2 + 8 * 16385
    assert case.algorithmic_bytes() == 1_081_896_032


def test_generators_are_pure_functions_of_their_seeds():
    a, b = wl.medium_norm("layernorm", rows=16), wl.medium_norm("layernorm", rows=16)
    assert torch.equal(a.x.view(torch.int16), b.x.view(torch.int16))
    assert torch.equal(a.gamma.view(torch.int16), b.gamma.view(torch.int16))
    r1 = wl.ragged_norm_backward("rmsnorm", rows=64, max_len=4096)
    r2 = wl.ragged_norm_backward("rmsnorm", rows=64, max_len=4096)
    assert torch.equal(r1.offsets, r2.offsets) and torch.equal(r1.dy.view(torch.int16),
                                                              r2.dy.view(torch.int16))
    assert not torch.equal(wl.ragged_lengths(64, 4096, wl._gen(4)),
                           wl.ragged_lengths(64, 4096, wl._gen(5)))


def test_every_case_is_consistent():
    for case in wl.all_cases(scale_down=256):
        assert case.algorithmic_bytes() > 0, case.name
        if case.ragged:
            off = case.offsets.numpy()
            assert off[0] == 0 and np.all(np.diff(off) >= 0) and off[-1] == case.x.numel()
            assert np.diff(off).max() <= case.max_len
            if case.gamma is not None:
                assert case.gamma.numel() >= case.max_len
        elif case.gamma is not None:
            assert case.gamma.numel() == case.x.shape[1]
        if case.dy is not None:
            assert case.dy.shape == case.x.shape and case.op.endswith("_backward")
