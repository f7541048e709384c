"""Windowed 3D attention: CUDA path vs the fp64 oracle (GB300 only).

A query attends the keys inside its kt x kh x kw window on the (t, h, w)
token grid (appendix Table 4 of the vidax paper: the LTX-2.5 VAE decoder's
neighbourhood attention).  The kernel takes query tiles as 3-D bricks of the
grid and key tiles as 3-D boxes over each unit's window union, shapes chosen
per grid.  Cases: both border rules, D = 64 and 128, grid sides that no
brick or box side divides (bricks and boxes reaching past the grid), axes of
length 1, a single token, windows larger than the grid, a 1 x 1 x 1 window,
more units than the persistent grid has CTAs, and a grid of 32760 tokens.
"""
import math

import pytest
import torch

from parity import compare, run_gpu, run_oracle

from paper_2609_18077_gb300 import workloads

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_18077_gb300 import build, binding
    build.build()
    binding.load()


CASES = [
    # B, H, D, grid, window, neighbourhood
    (1, 2, 128, (4, 6, 9), (3, 3, 3), True),
    (1, 2, 128, (4, 6, 9), (3, 3, 3), False),
    (2, 1, 64, (3, 8, 50), (3, 5, 11), True),      # rows of 50 keys: tiles span row borders
    (1, 2, 64, (5, 4, 300), (1, 3, 21), False),    # one row spans several tiles
    (1, 1, 128, (2, 3, 4), (3, 5, 7), True),       # window larger than the grid: dense
    (1, 2, 128, (3, 5, 7), (1, 1, 1), True),       # only the query's own key
    (2, 4, 128, (6, 12, 20), (5, 5, 5), True),     # 1440 tokens x 8 heads: more units than CTAs
    (2, 2, 128, (7, 1, 300), (3, 1, 5), False),    # an axis of length 1, a long ragged row
    (1, 1, 64, (1, 1, 1), (1, 1, 1), True),        # a single token
    (1, 3, 128, (9, 17, 23), (5, 3, 7), True),     # every side ragged against bricks and boxes
    (1, 2, 128, (21, 30, 52), (11, 11, 11), True),  # small480's grid with the decoder's window
    # 156 units: every persistent CTA takes one, four take a second
    (1, 13, 128, (8, 16, 24), (5, 5, 5), True),
    (1, 13, 64, (8, 16, 24), (7, 3, 5), False),
]


@pytest.mark.parametrize("B,H,D,grid,window,nb", CASES)
def test_window_cases(B, H, D, grid, window, nb):
    S = grid[0] * grid[1] * grid[2]
    q, k, v = workloads.random_qkv(B, H, S, S, D, seed=900 + S + D, logit_gain=1.5)
    win = (grid, window, nb)
    out, lse = run_gpu(q, k, v, 1 / math.sqrt(D), window=win)
    o_ref, lse_ref = run_oracle(q, k, v, 1 / math.sqrt(D), window=win)
    stats = compare(out, lse, o_ref, lse_ref)
    print(f"{grid} {window} nb={nb}: O max {stats[0]:.3e} mean {stats[1]:.3e} LSE rel {stats[2]:.3e}")


def test_window_whole_grid_equals_dense_attention():
    """A neighbourhood window spanning the grid is dense attention: the window
    kernel (every key box of the grid visited, in box order) and the dense
    kernel (key tiles in raster order) both match the oracle's dense result."""
    grid, D = (4, 8, 8), 128
    S = 256
    q, k, v = workloads.random_qkv(1, 3, S, S, D, seed=77, logit_gain=1.5)
    o1, l1 = run_gpu(q, k, v, 1 / math.sqrt(D), window=(grid, (5, 9, 9), True))
    o2, l2 = run_gpu(q, k, v, 1 / math.sqrt(D))
    o_ref, l_ref = run_oracle(q, k, v, 1 / math.sqrt(D))
    compare(o1, l1, o_ref, l_ref)
    compare(o2, l2, o_ref, l_ref)
