"""Windowed 3D attention: CUDA path vs the fp64 oracle (GB300 only).

A query attends the keys inside its kt x kh x kw window on the (t, h, w)
token grid (appendix Table 4 of the vidax paper: the LTX-2.5 VAE decoder's
neighbourhood attention).  Cases: both border rules, D = 64 and 128, grids
whose token count is not a multiple of the 128-token tile, rows of one and of
many tiles, windows larger than the grid, a 1 x 1 x 1 window and more units
than the persistent grid has CTAs.
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


def test_window_whole_grid_equals_dense_kernel():
    """A neighbourhood window spanning the grid visits every key tile; it equals the
    dense kernel to within the attention tolerance (tile masks only add -inf logits
    past the sequence end, which the dense kernel masks too)."""
    grid, D = (4, 8, 8), 128
    S = 256
    q, k, v = workloads.random_qkv(1, 3, S, S, D, seed=77, logit_gain=1.5)
    o1, l1 = run_gpu(q, k, v, 1 / math.sqrt(D), window=(grid, (5, 9, 9), True))
    o2, l2 = run_gpu(q, k, v, 1 / math.sqrt(D))
    assert torch.equal(o1.view(torch.int16), o2.view(torch.int16))
    assert torch.equal(l1, l2)
