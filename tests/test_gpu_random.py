"""Seeded random sweep: the CUDA path against the fp64 oracle on drawn shapes (GB300 only).

The other GPU tests pick their cases by hand, at tile borders and the edge
cases each problem kind has.  This sweep draws 98 more from one fixed seed,
across every kind, so that combinations nobody picked are compared too:
- dense, any lengths and both head dims, negative scales;
- dense calls whose short last round is split along the keys (the head
  count is chosen from the device's multiprocessor count);
- padded text, lengths anywhere in [0, Skv] over NaN padding;
- segment ids in runs, ids repeated across runs;
- windowed 3D attention, both border rules, windows up to larger than the
  grid.
Each case is compared element by element at the fixed tolerances.
"""
import math

import numpy as np
import pytest
import torch

from parity import check_case, compare, run_gpu, run_oracle

from paper_2609_18077_gb300 import workloads

pytestmark = pytest.mark.gpu

SEED = 20261202


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_18077_gb300 import build, binding
    build.build()
    binding.load()


def _rng(kind):
    return np.random.default_rng([SEED, kind])


def _scale(rng, D):
    s = float(rng.uniform(0.5, 1.5)) / math.sqrt(D)
    return -s if rng.random() < 0.15 else s


def _dense_cases():
    rng = _rng(1)
    out = []
    for i in range(30):
        D = int(rng.choice([64, 128]))
        out.append((int(rng.integers(1, 4)), int(rng.integers(1, 6)), int(rng.integers(1, 1401)),
                    int(rng.integers(1, 1401)), D, _scale(rng, D), float(rng.choice([1.0, 1.7, 3.0])), 100 + i))
    return out


@pytest.mark.parametrize("B,H,Sq,Skv,D,scale,gain,seed", _dense_cases())
def test_random_dense(B, H, Sq, Skv, D, scale, gain, seed):
    check_case(B, H, Sq, Skv, D, scale, seed, gain)


def _split_cases():
    rng = _rng(2)
    return [(int(rng.choice([64, 128])), int(rng.integers(600, 1101)), int(rng.integers(1, 40)), 200 + i)
            for i in range(8)]


@pytest.mark.parametrize("D,Sq,extra,seed", _split_cases())
def test_random_split_tail(D, Sq, extra, seed):
    """units = H * ceil(Sq / 256) just past one full round of CTAs: the dense
    kernel cuts the short last round's units along the keys."""
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    pairs = math.ceil(Sq / 256)
    H = (sms + extra + pairs - 1) // pairs   # at least sms + extra units
    rows = workloads.draw_rows(1, H, Sq, 32, seed)
    check_case(1, H, Sq, Sq, D, 1 / math.sqrt(D), seed, 1.0, rows=rows)


def _varlen_cases():
    rng = _rng(3)
    out = []
    for i in range(20):
        B, Skv = int(rng.integers(1, 6)), int(rng.integers(1, 801))
        lens = [int(x) for x in rng.integers(0, Skv + 1, size=B)]
        lens[0] = int(rng.choice([0, Skv, lens[0]]))
        D = int(rng.choice([64, 128]))
        out.append((B, int(rng.integers(1, 5)), int(rng.integers(1, 901)), Skv, D, lens, 300 + i))
    return out


@pytest.mark.parametrize("B,H,Sq,Skv,D,lens,seed", _varlen_cases())
def test_random_varlen(B, H, Sq, Skv, D, lens, seed):
    check_case(B, H, Sq, Skv, D, 1 / math.sqrt(D), seed, 1.0, kv_lens=np.array(lens, np.int32))


def _segment_ids(rng, B, S):
    ids = np.empty((B, S), np.int32)
    for b in range(B):
        cuts = np.sort(rng.choice(np.arange(1, S), size=min(int(rng.integers(0, 6)), S - 1), replace=False)) \
            if S > 1 else np.array([], np.int64)
        bounds = [0, *cuts.tolist(), S]
        for lo, hi in zip(bounds[:-1], bounds[1:]):
            ids[b, lo:hi] = int(rng.integers(0, 4))   # ids may repeat across runs
    return ids


def _segment_cases():
    rng = _rng(4)
    out = []
    for i in range(20):
        B, S = int(rng.integers(1, 4)), int(rng.integers(2, 901))
        out.append((B, int(rng.integers(1, 4)), S, int(rng.choice([64, 128])), _segment_ids(rng, B, S), 400 + i))
    return out


@pytest.mark.parametrize("B,H,S,D,ids,seed", _segment_cases())
def test_random_segments(B, H, S, D, ids, seed):
    check_case(B, H, S, S, D, 1 / math.sqrt(D), seed, 1.5, q_seg=ids, kv_seg=ids)


def _window_cases():
    rng = _rng(5)
    out = []
    for i in range(20):
        grid = (int(rng.integers(1, 9)), int(rng.integers(1, 21)), int(rng.integers(1, 41)))
        window = tuple(int(2 * rng.integers(0, 8) + 1) for _ in range(3))
        out.append((int(rng.integers(1, 3)), int(rng.integers(1, 4)), int(rng.choice([64, 128])), grid, window,
                    bool(rng.random() < 0.5), 500 + i))
    return out


@pytest.mark.parametrize("B,H,D,grid,window,nb", [c[:6] for c in _window_cases()])
def test_random_window(B, H, D, grid, window, nb):
    S = grid[0] * grid[1] * grid[2]
    q, k, v = workloads.random_qkv(B, H, S, S, D, seed=500 + S + D, logit_gain=1.5)
    win = (grid, window, nb)
    out, lse = run_gpu(q, k, v, 1 / math.sqrt(D), window=win)
    o_ref, lse_ref = run_oracle(q, k, v, 1 / math.sqrt(D), window=win)
    compare(out, lse, o_ref, lse_ref)
