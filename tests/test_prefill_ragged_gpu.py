"""Persistent prefill on ragged lengths with several units per block, against the fp64 oracle
(needs a GB300).

These shapes give every block a first unit whose key tiles are all issued by the MMA warp's
first two S products (at most two key tiles), followed by short units: the length is not a
multiple of the 128-row tile, so the last query tile is partial and the heaviest unit has two
key tiles.  When the MMA warp issued those first two S products from a separate prologue, the
key-tile count it took over from there for the block's second unit was 0 in the main loop, and
the warp waited for a key tile that no role produces (the blocks' bounded waits gave up after
2 s and the call reported FAV_ERR_DEVICE_TIMEOUT).  Every case here compares every output row
with the oracle and checks that no bounded wait gave up (run_gpu asserts a zero device
status)."""
import numpy as np
import pytest

import paper_2608_18656_gb300 as fav
from paper_2608_18656_gb300 import inputs as I
from gpu_util import check, run_gpu
import test_varlen_gpu as V

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _reset():
    fav.set_path(fav.PATH_AUTO)
    fav.set_prefill_grid(0)
    yield
    fav.set_path(fav.PATH_AUTO)
    fav.set_prefill_grid(0)


def W(dtype, B, Hq, Hkv, N, D, causal=True, seed=0):
    return I.Workload("ragged", dtype, B, Hq, Hkv, N, N, D, causal, False, seed)


def run_check(w, grid):
    fav.set_prefill_grid(grid)
    x = I.make_inputs(w)
    o, lse = run_gpu(w, x)
    assert fav.last_path() == fav.PATH_PREFILL
    check(w, o, lse, x)


def test_capped_grid_reproducer():
    """B 1, Hq 8, Hkv 2, N 200, fp16, causal on 7 blocks: blocks 2-6 own a two-tile unit then a
    one- or two-tile unit (the case that stopped at a bounded wait)."""
    run_check(W(I.F16, 1, 8, 2, 200, 128, seed=1), 7)


@pytest.mark.parametrize("dtype", [I.F16, I.BF16])
@pytest.mark.parametrize("B,Hq,Hkv", [(16, 8, 2), (8, 32, 32)])
def test_default_grid_two_units_per_block(dtype, B, Hq, Hkv):
    """256 or 512 query tiles of 200-row sequences on one block per SM: most blocks take two
    units, the first with two key tiles."""
    run_check(W(dtype, B, Hq, Hkv, 200, 128, seed=B + Hq), 0)


@pytest.mark.parametrize("N", [130, 200, 257, 385])
@pytest.mark.parametrize("grid", [0, 2, 3, 5, 7])
def test_ragged_lengths_and_grids(N, grid):
    """Lengths one past, or between, multiples of the tile, on grids of 2 to 7 blocks and the
    default grid (2 to 16 units per block)."""
    run_check(W(I.F16, 2, 4, 1, N, 128, seed=N + grid), grid)


@pytest.mark.parametrize("grid", [0, 3, 7])
def test_ragged_non_causal(grid):
    run_check(W(I.BF16, 3, 8, 2, 200, 128, causal=False, seed=grid), grid)


@pytest.mark.parametrize("grid", [0, 7])
@pytest.mark.parametrize("D", [128, 64])
def test_ragged_head_dim_64_and_128_bf16(D, grid):
    """The same ragged shape on both prefill kernels (D = 64 is the two-tile kernel)."""
    run_check(W(I.BF16, 4, 8, 2, 200, D, seed=D + grid), grid)


@pytest.mark.parametrize("grid", [0, 3, 7])
@pytest.mark.parametrize("D", [128, 64])
def test_varlen_ragged_short_units(D, grid):
    """Packed batch whose sequences end inside a tile (200, 130, 70, 256, 1 and 129 tokens):
    the packed-batch form of the shapes above."""
    fav.set_prefill_grid(grid)
    lens = [200, 130, 70, 256, 1, 129]
    q, k, v, cq, ck = V.packed(I.F16, lens, lens, 8, 2, D, seed=D + grid)
    scale = float(np.float32(1.0 / np.sqrt(D)))
    o, lse = V.run(I.F16, q, k, v, cq, ck, True, scale)
    V.check(q, k, v, cq, ck, o, lse, I.F16, True, scale)
