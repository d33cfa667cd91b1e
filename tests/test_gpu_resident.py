"""The register-resident tile designs against the staged tile design.

All cut a MEDIUM or LARGE row into the same 1 KiB tiles, reduce each tile in
the same order and combine the tile partials in the same fixed order; the
resident designs only keep a lane's chunks in registers instead of reading
the staged row three times.  So they must agree bit for bit on every shape
they can take:
  * the whole-tile kernel (the default for dense MEDIUM rows that are a
    whole number of tiles): one CTA per row of 8, 16 or 32 tiles, and, with
    ROWOP_RESIDENT=2, cluster splits of LARGE rows into equal portions;
  * the streamed split of LARGE rows (each cluster portion read twice
    through a ring of pieces, the default for whole-block portions).
Parity of every design against the oracle is checked here as well.
"""
import os

import pytest
import torch

from tests.gpu_util import DTYPE_IDS, ALL_OPS, DTYPES, ESIZE
from tests.test_gpu_dense import run_case

pytestmark = pytest.mark.gpu

KNOBS = ("ROWOP_RESIDENT", "ROWOP_FORCE_BUCKET", "ROWOP_CLUSTER", "ROWOP_STAGES", "ROWOP_STREAM")


@pytest.fixture(scope="module")
def rw():
    from paper_2607_23089_gb300 import build, rowop
    build.build()
    rowop.load()
    torch.cuda.set_device(0)
    return rowop


def _run(rw, op, dtype, rows, cols, resident, ld=None, x_off=0, bucket=None, cluster=None,
         stages=None, affine=True, check=False):
    old = {k: os.environ.get(k) for k in KNOBS}
    try:
        os.environ["ROWOP_RESIDENT"] = str(int(resident))
        os.environ["ROWOP_STREAM"] = "0"  # the streamed split has its own tests below
        for k, v in (("ROWOP_FORCE_BUCKET", bucket), ("ROWOP_CLUSTER", cluster),
                     ("ROWOP_STAGES", stages)):
            if v is not None:
                os.environ[k] = str(v)
            else:
                os.environ.pop(k, None)
        return run_case(rw, op, dtype, rows, cols, ld=ld, x_off=x_off, y_off=x_off,
                        seed=cols + rows, affine=affine, check=check).clone()
    finally:
        for k, v in old.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v


def _bits(t):
    return t.view(torch.int32) if t.dtype == torch.float32 else t.view(torch.int16)


# whole-tile rows: (cols per dtype size, design): MEDIUM rows of 8, 16 and 32
# tiles on one CTA; LARGE rows split into equal portions
FULL_MEDIUM = {4: (2048, 4096, 8192), 2: (4096, 8192, 16384)}
FULL_LARGE = {4: ((32768, 3), (65536, 3), (262144, 2)), 2: ((65536, 3), (131072, 3))}


@pytest.mark.parametrize("dtype", DTYPES, ids=DTYPE_IDS)
@pytest.mark.parametrize("op", ALL_OPS)
def test_whole_tile_medium_equals_staged(rw, op, dtype):
    for cols in FULL_MEDIUM[ESIZE[dtype]]:
        for rows in (1, 37, 700):
            a = _run(rw, op, dtype, rows, cols, 1, check=True)
            b = _run(rw, op, dtype, rows, cols, 0)
            assert torch.equal(_bits(a), _bits(b)), (cols, rows)
    # a row stride of whole chunks wider than the row
    a = _run(rw, op, dtype, 9, FULL_MEDIUM[ESIZE[dtype]][0], 1,
             ld=FULL_MEDIUM[ESIZE[dtype]][0] + 64, check=True)
    b = _run(rw, op, dtype, 9, FULL_MEDIUM[ESIZE[dtype]][0], 0,
             ld=FULL_MEDIUM[ESIZE[dtype]][0] + 64)
    assert torch.equal(_bits(a), _bits(b))


@pytest.mark.parametrize("dtype", DTYPES, ids=DTYPE_IDS)
@pytest.mark.parametrize("op", ALL_OPS)
def test_whole_tile_large_equals_staged(rw, op, dtype):
    for cols, rows in FULL_LARGE[ESIZE[dtype]]:
        a = _run(rw, op, dtype, rows, cols, 2, check=True)
        b = _run(rw, op, dtype, rows, cols, 0)
        assert torch.equal(_bits(a), _bits(b)), cols


@pytest.mark.parametrize("op", ("layernorm", "rmsnorm"))
def test_whole_tile_without_affine(rw, op):
    for dtype in (torch.float32, torch.bfloat16):
        cols = FULL_MEDIUM[ESIZE[dtype]][0]
        a = _run(rw, op, dtype, 9, cols, 1, affine=False, check=True)
        b = _run(rw, op, dtype, 9, cols, 0, affine=False)
        assert torch.equal(_bits(a), _bits(b))


@pytest.mark.parametrize("stages", [1, 2, 5])
def test_whole_tile_stage_counts(rw, stages):
    """Refilling a stage right after the row's barrier is safe at any ring
    depth: one stage (every row waits for its own copy) to several."""
    for op in ("layernorm", "softmax"):
        a = _run(rw, op, torch.bfloat16, 301, 4096, 1, stages=stages, check=True)
        b = _run(rw, op, torch.bfloat16, 301, 4096, 0)
        assert torch.equal(_bits(a), _bits(b))


# LARGE rows whose cluster portions are whole 64-tile blocks: (cols per dtype
# size, rows) -- the streamed split against the staged split
STREAM_LARGE = {4: ((32768, 5), (262144, 3)), 2: ((65536, 5), (131072, 3))}


def _run_knobs(rw, op, dtype, rows, cols, knobs, check=False):
    names = ("ROWOP_STREAM", "ROWOP_CLUSTER", "ROWOP_STAGES", "ROWOP_CTAS_PER_SM", "ROWOP_RESIDENT")
    old = {k: os.environ.get(k) for k in names}
    try:
        for k in names:
            os.environ.pop(k, None)
        os.environ.update({k: str(v) for k, v in knobs.items()})
        return run_case(rw, op, dtype, rows, cols, seed=cols + rows, check=check).clone()
    finally:
        for k, v in old.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v


@pytest.mark.parametrize("dtype", DTYPES, ids=DTYPE_IDS)
@pytest.mark.parametrize("op", ALL_OPS)
def test_streamed_split_equals_staged(rw, op, dtype):
    """The streamed split (each portion read twice through a ring of pieces)
    forms the same tile partials, block partials and combine as the staged
    split, so the two agree bit for bit; checked against the oracle too."""
    for cols, rows in STREAM_LARGE[ESIZE[dtype]]:
        a = _run_knobs(rw, op, dtype, rows, cols, {"ROWOP_STREAM": 1}, check=True)
        b = _run_knobs(rw, op, dtype, rows, cols, {"ROWOP_STREAM": 0, "ROWOP_RESIDENT": 0})
        assert torch.equal(_bits(a), _bits(b)), cols


@pytest.mark.parametrize("knobs", [{"ROWOP_CLUSTER": 2}, {"ROWOP_CLUSTER": 8},
                                   {"ROWOP_CLUSTER": 16}, {"ROWOP_STAGES": 2},
                                   {"ROWOP_STAGES": 3}, {"ROWOP_CTAS_PER_SM": 1}],
                         ids=["cs2", "cs8", "cs16", "ring2", "ring3", "one_cta_sm"])
def test_streamed_split_shapes(rw, knobs):
    """Cluster sizes, ring depths (one that does not divide the pieces of a
    pass) and many rows per cluster (one CTA an SM): the same bits."""
    cols, rows = 262144, 40
    for op in ("logsoftmax", "layernorm"):
        a = _run_knobs(rw, op, torch.float32, rows, cols, dict(knobs, ROWOP_STREAM=1))
        b = _run_knobs(rw, op, torch.float32, rows, cols, {"ROWOP_STREAM": 0, "ROWOP_RESIDENT": 0})
        assert torch.equal(_bits(a), _bits(b)), knobs
