"""Seeded random sweep: the CUDA path against the fp64 oracle on drawn shapes (GB300 only).

The other GPU tests pick their cases by hand, at tile borders and the edge
cases each problem kind has.  This sweep draws 120 more from one fixed seed,
across every kind, so that combinations nobody picked are compared too:
- dense, any lengths and both head dims, negative scales;
- dense calls whose short last round is split along the keys (the head
  count is chosen from the device's multiprocessor count);
- padded text, lengths anywhere in [0, Skv] over NaN padding;
- segment ids in runs, ids repeated across runs;
- windowed 3D attention, both border rules, windows up to larger than the
  grid;
- the host-buffer entry points of every kind, chunk sizes drawn (0: the
  library's choice);
- the 3D RoPE on drawn grids, offsets, dimension splits, bases and pairings.
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


def _host_cases():
    rng = _rng(6)
    out = []
    for i in range(12):
        kind = ["dense", "varlen", "segments", "window"][i % 4]
        B, H, D = int(rng.integers(1, 4)), int(rng.integers(1, 5)), int(rng.choice([64, 128]))
        out.append((kind, B, H, D, int(rng.integers(0, B * H + 1)), 600 + i))
    return out


@pytest.mark.parametrize("kind,B,H,D,chunk_rows,seed", _host_cases())
def test_random_host_buffers(kind, B, H, D, chunk_rows, seed):
    """The host-buffer entry points (chunk_rows 0: the library's choice) against the oracle."""
    from paper_2609_18077_gb300 import binding
    rng = np.random.default_rng([SEED, seed])
    scale = 1 / math.sqrt(D)
    lens = q_seg = window = None
    if kind == "window":
        grid = (int(rng.integers(1, 6)), int(rng.integers(1, 13)), int(rng.integers(1, 25)))
        window = (grid, tuple(int(2 * rng.integers(0, 6) + 1) for _ in range(3)), bool(rng.random() < 0.5))
        Sq = Skv = grid[0] * grid[1] * grid[2]
    else:
        Sq = int(rng.integers(1, 700))
        Skv = Sq if kind == "segments" else int(rng.integers(1, 700))
    q, k, v = workloads.random_qkv(B, H, Sq, Skv, D, seed, 1.5)
    if kind == "varlen":
        lens = rng.integers(0, Skv + 1, size=B).astype(np.int32)
        k, v = workloads.pad_invalid_keys(k, v, lens)
    if kind == "segments":
        q_seg = _segment_ids(rng, B, Sq)
    qp, kp, vp = (t.pin_memory() for t in (q, k, v))
    if kind == "window":
        out, lse = binding.attn_fwd_win3d_host(qp, kp, vp, window[0], window[1], window[2], scale=scale,
                                               chunk_rows=chunk_rows)
    elif kind == "segments":
        segs = torch.from_numpy(q_seg)
        out, lse = binding.attn_fwd_segments_host(qp, kp, vp, segs, segs, scale=scale, chunk_rows=chunk_rows)
    else:
        out, lse = binding.attn_fwd_host(qp, kp, vp, kv_lens=None if lens is None else torch.from_numpy(lens),
                                         scale=scale, chunk_rows=chunk_rows)
    assert binding.check_device_error() == binding.VDX_OK
    o_ref, lse_ref = run_oracle(q, k, v, scale, lens, q_seg=q_seg, kv_seg=q_seg, window=window)
    compare(out, lse, o_ref, lse_ref)


def _rope_cases():
    rng = _rng(7)
    out = []
    for i in range(10):
        D = int(rng.choice([64, 96, 128]))
        inter = bool(rng.random() < 0.6)
        dims = sorted(2 * rng.integers(0, D // 6 + 1, size=3))   # each even, summing to at most D
        dims = tuple(int(d) for d in rng.permutation(dims))
        grid = (int(rng.integers(1, 7)), int(rng.integers(1, 12)), int(rng.integers(1, 20)))
        out.append((int(rng.integers(1, 3)), int(rng.integers(1, 4)), D, grid, int(rng.integers(0, 9)),
                    int(rng.integers(0, 9)), dims, float(rng.choice([10.0, 500.0, 1e4])), inter, 700 + i))
    return out


@pytest.mark.parametrize("B,H,D,grid,s0,after,dims,theta,inter,seed", _rope_cases())
def test_random_rope(B, H, D, grid, s0, after, dims, theta, inter, seed):
    """vdx_rope3d against the oracle's rotation: within 2^-8 of each output
    (its bf16 rounding) plus 2e-5 of the row's largest input (the fp32 angle)."""
    import oracle
    from paper_2609_18077_gb300 import binding
    S = s0 + grid[0] * grid[1] * grid[2] + after
    x, _, _ = workloads.random_qkv(B, H, S, 1, D, seed, 1.5)
    y_ref = oracle.rope3d(workloads.bf16_bits(x), grid, s0, dims, theta, inter)
    y = binding.rope3d(x.cuda(), grid, s0, dims, theta, inter)
    assert binding.check_device_error() == binding.VDX_OK
    yd = y.float().double().cpu().numpy()
    bound = 2.0 ** -8 * np.abs(y_ref) + 2e-5 * np.max(np.abs(x.float().double().numpy()), axis=-1, keepdims=True)
    assert np.all(np.isfinite(yd)) and np.all(np.abs(yd - y_ref) <= bound)
