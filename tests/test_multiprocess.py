"""The multi-rank path on the CPU: world size 2 over gloo.

Rows are independent, so several GPUs run replicas with no collective on the
data path; the only inter-rank steps are a barrier around the timed region and
a max over ranks of the measured time.  These tests run those steps with two
gloo ranks (no GPU), launch the reference arm under torch.distributed.run as
the benchmark driver does (rank 0 alone prints one JSON line), and check the
row partition a batch is split by (paper_2607_23089_gb300.shard): blocks that
tile the batch, balanced, each a batch of its own whose results put together
equal the whole batch's.
"""
import json
import os
import socket
import subprocess
import sys

import numpy as np
import pytest
import torch.multiprocessing as mp

from paper_2607_23089_gb300 import shard

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    import torch
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        bench.barrier(world)
        # each rank's own time; every rank must get the largest
        got = bench.max_over_ranks(1.5 + rank, world, torch.device("cpu"))
        bench.barrier(world)
        out[rank] = got
    finally:
        dist.destroy_process_group()


def test_barrier_and_max_over_ranks_gloo():
    world = 2
    port = _free_port()
    out = mp.Manager().dict()
    mp.spawn(_rank_main, args=(world, port, out), nprocs=world, join=True)
    assert dict(out) == {0: 2.5, 1: 2.5}


def test_reference_arm_under_torchrun():
    """`bench.py --impl reference` launched like the driver's N = 2 run: one
    JSON line, from rank 0, naming two GPUs; the other rank exits 0."""
    port = _free_port()
    env = dict(os.environ, ROWOP_REF_SAMPLE_ELEMS="300000")
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), "bench.py", "--impl",
           "reference", "--gpus", "2", "--steps", "1", "--warmup", "3"]
    r = subprocess.run(cmd, cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.strip().startswith("{")]
    assert len(lines) == 1, r.stdout
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2
    assert d["value"] > 0 and d["cpu_baseline"]["kind"] == "oracle"
    assert d["e2e"]["h2d_bytes_per_step"] == 0


def test_dense_blocks_tile_the_rows():
    for rows in (0, 1, 7, 8, 1000, 16385):
        for world in (1, 2, 3, 8):
            blocks = [shard.dense_block(rows, world, r) for r in range(world)]
            assert blocks[0][0] == 0 and blocks[-1][1] == rows
            assert all(a[1] == b[0] for a, b in zip(blocks, blocks[1:]))
            sizes = [hi - lo for lo, hi in blocks]
            assert max(sizes) - min(sizes) <= 1
    with pytest.raises(ValueError):
        shard.dense_block(10, 2, 2)


def test_ragged_blocks_tile_and_balance():
    rng = np.random.default_rng(5)
    cases = [np.zeros(1, np.int64), np.array([0, 0, 0], np.int64),
             np.array([0, 5], np.int64)]
    for n in (3, 50, 4000):
        lens = rng.integers(0, 3000, n)
        lens[rng.random(n) < 0.1] = 0
        cases.append(np.concatenate([[0], np.cumsum(lens)]).astype(np.int64) + 11)
    for off in cases:
        rows = off.shape[0] - 1
        total = int(off[-1] - off[0])
        longest = int(np.max(np.diff(off))) if rows else 0
        for world in (1, 2, 3, 8):
            blocks = [shard.ragged_block(off, world, r) for r in range(world)]
            assert blocks[0].row_lo == 0 and blocks[-1].row_hi == rows
            for a, b in zip(blocks, blocks[1:]):
                assert a.row_hi == b.row_lo and a.elem_hi == b.elem_lo
            for b in blocks:
                assert b.offsets[0] == 0 and b.offsets.shape[0] == b.rows + 1
                assert np.array_equal(b.offsets + b.elem_lo, off[b.row_lo:b.row_hi + 1])
                assert abs(b.elements - total / world) < max(longest, 1)
    with pytest.raises(ValueError):
        shard.ragged_cuts(np.array([0, 5, 3]), 2)


def _block_main(rank, world, port, out):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    from oracle import rowop_oracle as orc
    from paper_2607_23089_gb300 import shard as sh
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # every rank draws the same batch; each normalises its own block
        g = np.random.default_rng(3)
        lens = g.integers(0, 2000, 300)
        off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
        x = g.normal(0.0, 3.0, int(off[-1]))
        gam = g.normal(1.0, 0.1, 2000)
        b = sh.ragged_block(off, world, rank)
        y = orc.layernorm_ragged(x[b.elem_lo:b.elem_hi], b.offsets, gam, None, eps=1e-5)
        spans = [None] * world
        dist.all_gather_object(spans, (b.row_lo, b.row_hi, b.elem_lo, b.elem_hi))
        parts = [None] * world
        dist.all_gather_object(parts, y)
        if rank == 0:
            whole = orc.layernorm_ragged(x, off, gam, None, eps=1e-5)
            out["spans"] = spans
            out["equal"] = bool(np.array_equal(np.concatenate(parts), whole))
            out["rows"] = len(lens)
    finally:
        dist.destroy_process_group()


def test_ragged_blocks_over_two_gloo_ranks():
    """Each rank normalises its own block (no exchange on the data path); put
    together in rank order, the blocks' outputs equal the whole batch's, bit
    for bit."""
    world = 2
    port = _free_port()
    out = mp.Manager().dict()
    mp.spawn(_block_main, args=(world, port, out), nprocs=world, join=True)
    spans = out["spans"]
    assert spans[0][0] == 0 and spans[-1][1] == out["rows"] and spans[0][1] == spans[1][0]
    assert out["equal"]


if __name__ == "__main__":
    pytest.main([__file__, "-q"])
