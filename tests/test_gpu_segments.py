"""Joint attention with segment ids: CUDA path vs the fp64 oracle (GB300 only).

Query i of sample b attends key j iff q_seg[b, i] == kv_seg[b, j] (appendix
Table 4 of the vidax paper: padded text in joint text-video attention is
masked through segment ids that let the kernel skip key blocks).  The cases
cover the joint layout (text slots, then video), packed sequences, ids
interleaved at random, query segments that own no key (whole units and
single rows), Sq != Skv, ragged tails, negative and zero scales, and more
units than the persistent grid has CTAs.
"""
import math

import numpy as np
import pytest
import torch

from parity import check_case, run_gpu

from paper_2609_18077_gb300 import workloads

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_18077_gb300 import build, binding
    build.build()
    binding.load()


def _blocks(sizes, ids):
    return np.concatenate([np.full(n, i, np.int32) for n, i in zip(sizes, ids)])


def _joint(B, slots, video, lens):
    return workloads.joint_segments(np.array(lens, np.int32), slots, slots + video)


def _case(name):
    """(B, H, Sq, Skv, D, scale multiplier, q_seg, kv_seg)."""
    if name == "joint_text_first":
        seg = _joint(2, 100, 600, [37, 100])
        return 2, 2, 700, 700, 64, 1.0, seg, seg
    if name == "joint_text_first_d128":
        seg = _joint(2, 100, 600, [37, 1])
        return 2, 2, 700, 700, 128, 1.0, seg, seg
    if name == "joint_pad_on_tile_border":
        seg = _joint(2, 256, 300, [128, 5])
        return 2, 1, 556, 556, 128, 1.0, seg, seg
    if name == "packed":
        seg = _blocks([300, 129, 1, 570], [4, 7, 1, 2])[None].repeat(2, 0)
        seg[1] = _blocks([1000], [3])
        return 2, 2, 1000, 1000, 64, 1.0, seg, seg
    if name == "interleaved":
        rng = np.random.default_rng(40)
        qs = rng.integers(0, 3, size=(2, 300)).astype(np.int32)
        ks = rng.integers(0, 3, size=(2, 300)).astype(np.int32)
        return 2, 2, 300, 300, 64, 1.0, qs, ks
    if name == "absent_query_segment":
        ks = _blocks([400, 600], [1, 2])[None]
        qs = ks.copy()
        qs[0, 512:768] = 9      # a whole query-tile pair with no key: an empty list
        qs[0, 100] = -5         # one row with no key inside a visited tile
        return 1, 3, 1000, 1000, 128, 1.0, qs, ks
    if name == "cross_shaped":
        qs = _blocks([250, 250], [1, 2])[None].repeat(2, 0)
        ks = _blocks([100, 233], [1, 2])[None].repeat(2, 0)
        ks[1] = _blocks([333], [2])
        return 2, 2, 500, 333, 128, 1.0, qs, ks
    if name == "negative_scale":
        seg = _joint(1, 130, 400, [77])
        return 1, 2, 530, 530, 128, -1.0, seg, seg
    if name == "zero_scale":
        seg = _joint(1, 130, 400, [130])
        seg[0, 300:310] = 5
        return 1, 2, 530, 530, 64, 0.0, seg, seg
    if name == "many_units":
        seg = _joint(2, 226, 1774, [60, 200])
        return 2, 24, 2000, 2000, 64, 1.0, seg, seg
    raise KeyError(name)


CASES = ["joint_text_first", "joint_text_first_d128", "joint_pad_on_tile_border", "packed", "interleaved",
         "absent_query_segment", "cross_shaped", "negative_scale", "zero_scale", "many_units"]


@pytest.mark.parametrize("name", CASES)
def test_segments(name):
    B, H, Sq, Skv, D, smul, qs, ks = _case(name)
    stats = check_case(B, H, Sq, Skv, D, smul / math.sqrt(D), seed=500 + Sq + Skv + D, gain=1.5,
                       q_seg=qs, kv_seg=ks)
    print(f"{name}: O max {stats[0]:.3e} mean {stats[1]:.3e} LSE rel {stats[2]:.3e}")


@pytest.mark.parametrize("D", [64, 128])
def test_one_segment_is_the_dense_kernel(D):
    """A single id everywhere visits every tile unmasked: bit-identical to vdx_attn_fwd
    (the sizes keep the dense call on whole units: 24 units with 7 key tiles,
    too few for a cut of at least 8 tiles a part)."""
    B, H, S = 2, 3, 777
    q, k, v = workloads.random_qkv(B, H, S, S, D, seed=61 + D, logit_gain=1.5)
    seg = np.full((B, S), 42, np.int32)
    o1, l1 = run_gpu(q, k, v, 1 / math.sqrt(D), q_seg=seg, kv_seg=seg)
    o2, l2 = run_gpu(q, k, v, 1 / math.sqrt(D))
    assert torch.equal(o1.view(torch.int16), o2.view(torch.int16))
    assert torch.equal(l1, l2)
