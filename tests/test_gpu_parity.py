"""CUDA path vs the fp64 oracle, element by element, on seeded inputs (GB300 only)."""
import math

import numpy as np
import pytest
import torch

from parity import check_case, compare, run_gpu, run_oracle

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_18077_gb300 import build, binding
    build.build()
    binding.load()


# ragged sizes around the 128-row tile and the 256-row query-tile pair
EDGE = [
    # B, H, Sq, Skv, D, scale-multiplier (x 1/sqrt(D)), gain
    (1, 1, 1, 1, 64, 1.0, 1.0),
    (1, 1, 2, 2, 128, 1.0, 1.0),
    (1, 2, 63, 65, 64, 1.0, 1.0),
    (2, 1, 64, 64, 128, 1.0, 1.0),
    (1, 3, 65, 127, 128, 1.0, 1.0),
    (3, 1, 127, 128, 64, 1.0, 1.0),
    (1, 2, 128, 129, 128, 1.0, 1.7),
    (2, 2, 129, 192, 64, 1.0, 1.7),
    (1, 1, 192, 255, 128, 4.0, 1.0),
    (1, 2, 255, 257, 128, 1.0, 1.0),
    (2, 3, 257, 1000, 128, 1.0, 1.7),
    (1, 1, 1000, 63, 64, 1.0, 1.0),
    (1, 2, 384, 2, 128, 1.0, 1.0),
    (1, 1, 513, 1, 128, 1.0, 1.0),
    (2, 2, 300, 777, 64, 4.0, 1.7),
    (1, 1, 256, 256, 128, 0.0, 1.0),
    (1, 2, 200, 300, 128, -1.0, 1.0),
    (1, 1, 640, 3000, 128, 1.0, 3.0),
]


@pytest.mark.parametrize("B,H,Sq,Skv,D,smul,gain", EDGE)
def test_edge_shapes(B, H, Sq, Skv, D, smul, gain):
    check_case(B, H, Sq, Skv, D, smul / math.sqrt(D), seed=100 + Sq + 7 * Skv + D, gain=gain)


VARLEN = [
    # B, H, Sq, Skv_max, D, lens
    (3, 2, 200, 512, 128, [512, 64, 129]),
    (4, 1, 130, 300, 64, [0, 1, 299, 300]),
    (2, 2, 257, 128, 128, [127, 128]),
    (2, 1, 64, 1000, 128, [1000, 513]),
    (3, 1, 100, 256, 128, [-5, 9999, 255]),
]


@pytest.mark.parametrize("B,H,Sq,Skv,D,lens", VARLEN)
def test_varlen(B, H, Sq, Skv, D, lens):
    check_case(B, H, Sq, Skv, D, 1 / math.sqrt(D), seed=300 + Sq + Skv, kv_lens=np.array(lens, np.int32))


# Text cross-attention (padded text keys, per-sample lengths): lengths at
# every key-tile border (0, 1, 127/128/129, 255/256/257, 383/384/385,
# 511/512), short Skv_max, a single query row, and more work units than
# multiprocessors so that every persistent CTA walks several (b, h).
CROSS_EDGES = [0, 1, 127, 128, 129, 255, 256, 257, 300, 383, 384, 385, 511, 512]
CROSS = [
    # B, H, Sq, Skv_max, D, lens
    (len(CROSS_EDGES), 2, 300, 512, 128, CROSS_EDGES),
    (len(CROSS_EDGES), 2, 300, 512, 64, CROSS_EDGES),
    (3, 2, 129, 200, 128, [200, 57, 0]),
    (2, 3, 1, 256, 64, [256, 100]),
    (4, 40, 640, 512, 128, [223, 215, 512, 300]),
    (2, 48, 384, 512, 64, [0, 171]),
]


@pytest.mark.parametrize("B,H,Sq,Skv,D,lens", CROSS)
def test_text_cross_attention(B, H, Sq, Skv, D, lens):
    check_case(B, H, Sq, Skv, D, 1 / math.sqrt(D), seed=600 + B * H + Sq, gain=1.5,
               kv_lens=np.array(lens, np.int32))


@pytest.mark.parametrize("smul,gain", [(-1.0, 1.5), (0.0, 1.0), (4.0, 3.0)])
def test_text_cross_attention_scales(smul, gain):
    """Negative and zero logit scales, and logits spread wide enough that a
    later key tile's maximum moves past the lazy-rescale threshold."""
    lens = np.array([512, 300, 257, 40], np.int32)
    check_case(4, 3, 260, 512, 128, smul / math.sqrt(128), seed=700, gain=gain, kv_lens=lens)


def test_text_cross_attention_canaries_and_determinism():
    """The varlen instance's TMA stores of O stay inside out (ragged Sq: the
    last tile is clipped), LSE inside lse; two calls give the same bits."""
    from paper_2609_18077_gb300 import binding, workloads
    B, H, Sq, Skv, D = 3, 5, 200, 512, 128
    lens = np.array([512, 129, 0], np.int32)
    q, k, v = workloads.random_qkv(B, H, Sq, Skv, D, seed=11)
    k, v = workloads.pad_invalid_keys(k, v, lens)
    q, k, v = q.cuda(), k.cuda(), v.cuda()
    ld = torch.from_numpy(lens).cuda()
    pad = 4096
    obuf = torch.full((pad + B * H * Sq * D + pad,), float("nan"), dtype=torch.bfloat16, device="cuda")
    lbuf = torch.full((pad + B * H * Sq + pad,), float("nan"), dtype=torch.float32, device="cuda")
    out = obuf[pad:pad + B * H * Sq * D].view(B, H, Sq, D)
    lse = lbuf[pad:pad + B * H * Sq].view(B, H, Sq)
    binding.attn_fwd_varlen(q, k, v, ld, scale=D ** -0.5, out=out, lse=lse)
    assert binding.check_device_error() == binding.VDX_OK
    assert torch.isnan(obuf[:pad]).all() and torch.isnan(obuf[-pad:]).all()
    assert torch.isnan(lbuf[:pad]).all() and torch.isnan(lbuf[-pad:]).all()
    assert torch.isfinite(out).all()
    assert torch.isneginf(lse[2]).all() and torch.isfinite(lse[:2]).all()
    o2, l2 = binding.attn_fwd_varlen(q, k, v, ld, scale=D ** -0.5)
    assert torch.equal(out.view(torch.int16), o2.view(torch.int16)) and torch.equal(lse, l2)


def test_varlen_long_text_many_units():
    """Long padded key sequences with mixed lengths over many units (key
    tiles skipped past each sample's length)."""
    lens = np.array([0, 600, 1, 513, 129, 0, 256, 599], np.int32)
    check_case(8, 20, 257, 600, 128, 128 ** -0.5, seed=502, kv_lens=lens)


def test_tiny_workload_full():
    from paper_2609_18077_gb300 import workloads
    w = workloads.generate("tiny")
    out, lse = run_gpu(w["q"], w["k"], w["v"], w["scale"])
    o_ref, lse_ref = run_oracle(w["q"], w["k"], w["v"], w["scale"])
    compare(out, lse, o_ref, lse_ref)


def test_lse_optional():
    from paper_2609_18077_gb300 import workloads
    q, k, v = workloads.random_qkv(1, 2, 300, 200, 128, seed=5)
    out, lse = run_gpu(q, k, v, 0.1, with_lse=False)
    assert lse is None
    o_ref, _ = run_oracle(q, k, v, 0.1)
    compare(out, None, o_ref, None)


def test_deterministic():
    from paper_2609_18077_gb300 import workloads
    q, k, v = workloads.random_qkv(2, 3, 700, 900, 128, seed=6, logit_gain=1.7)
    o1, l1 = run_gpu(q, k, v, 128 ** -0.5)
    o2, l2 = run_gpu(q, k, v, 128 ** -0.5)
    assert torch.equal(o1, o2) and torch.equal(l1, l2)


def test_guard_canaries():
    """Writes stay inside out/lse: NaN-filled margins around both are untouched."""
    from paper_2609_18077_gb300 import binding, workloads
    B, H, Sq, Skv, D = 1, 2, 200, 130, 128
    q, k, v = (t.cuda() for t in workloads.random_qkv(B, H, Sq, Skv, D, seed=7))
    pad = 4096
    obuf = torch.full((pad + B * H * Sq * D + pad,), float("nan"), dtype=torch.bfloat16, device="cuda")
    lbuf = torch.full((pad + B * H * Sq + pad,), float("nan"), dtype=torch.float32, device="cuda")
    out = obuf[pad:pad + B * H * Sq * D].view(B, H, Sq, D)
    lse = lbuf[pad:pad + B * H * Sq].view(B, H, Sq)
    binding.attn_fwd(q, k, v, scale=D ** -0.5, out=out, lse=lse)
    assert binding.check_device_error() == binding.VDX_OK
    assert torch.isnan(obuf[:pad]).all() and torch.isnan(obuf[-pad:]).all()
    assert torch.isnan(lbuf[:pad]).all() and torch.isnan(lbuf[-pad:]).all()
    assert torch.isfinite(out).all() and torch.isfinite(lse).all()


def test_head_partition_equivalence():
    """Heads are independent: one call equals per-head-slice calls (a 1-GPU stand-in
    for the head-sharded layout a multi-GPU run would use)."""
    from paper_2609_18077_gb300 import workloads
    q, k, v = workloads.random_qkv(1, 4, 400, 500, 128, seed=8)
    o, l = run_gpu(q, k, v, 0.09)
    for h0 in (0, 2):
        oh, lh = run_gpu(q[:, h0:h0 + 2].contiguous(), k[:, h0:h0 + 2].contiguous(),
                         v[:, h0:h0 + 2].contiguous(), 0.09)
        assert torch.equal(oh, o[:, h0:h0 + 2]) and torch.equal(lh, l[:, h0:h0 + 2])


def test_timeout_selftest_reports_and_recovers():
    """A bounded wait that nothing satisfies reports VDX_ERR_TIMEOUT; the context stays usable."""
    from paper_2609_18077_gb300 import binding
    assert binding.check_device_error() == binding.VDX_OK
    assert binding.selftest_wait_timeout(20000) == binding.VDX_OK
    assert binding.check_device_error() == binding.VDX_ERR_TIMEOUT
    assert binding.check_device_error() == binding.VDX_OK
    check_case(1, 1, 130, 140, 64, 0.125, seed=9)


# More work units (b*h x query-tile pairs) than multiprocessors, so every
# persistent CTA walks several units and the K/V stream crosses unit borders.
MULTI_UNIT = [
    # B, H, Sq, Skv, D
    (1, 100, 300, 200, 128),
    (2, 90, 513, 129, 64),
    (3, 60, 256, 1, 128),
]


@pytest.mark.parametrize("B,H,Sq,Skv,D", MULTI_UNIT)
def test_many_units_per_cta(B, H, Sq, Skv, D):
    check_case(B, H, Sq, Skv, D, 1 / math.sqrt(D), seed=400 + H + Skv, gain=1.4)


def test_varlen_many_units_mixed_lengths():
    """Samples with no keys, one key, ragged and full tiles interleaved across
    the units every CTA walks."""
    lens = np.array([0, 300, 1, 129, 0, 256, 64, 255], np.int32)
    check_case(8, 20, 257, 300, 128, 128 ** -0.5, seed=501, kv_lens=lens)


# A short last round: with 152 SMs these leave 2 and 8 units for the last
# round, which the library splits along the keys into parts on idle CTAs and
# merges through its workspace (16 parts of one key tile, 8 parts with a
# ragged last key tile).
SPLIT_TAIL = [
    # B, H, Sq, Skv, D
    (1, 154, 256, 2000, 128),
    (2, 80, 100, 1000, 64),
    (1, 153, 200, 300, 128),
]


@pytest.mark.parametrize("B,H,Sq,Skv,D", SPLIT_TAIL)
def test_split_tail(B, H, Sq, Skv, D):
    check_case(B, H, Sq, Skv, D, 1 / math.sqrt(D), seed=600 + H + Skv, gain=1.6)


def test_split_tail_deterministic_and_lse_optional():
    from paper_2609_18077_gb300 import workloads
    q, k, v = workloads.random_qkv(1, 154, 256, 2000, 128, seed=7, logit_gain=1.6)
    o1, l1 = run_gpu(q, k, v, 128 ** -0.5)
    o2, l2 = run_gpu(q, k, v, 128 ** -0.5)
    assert torch.equal(o1, o2) and torch.equal(l1, l2)
    o3, l3 = run_gpu(q, k, v, 128 ** -0.5, with_lse=False)
    assert l3 is None and torch.equal(o3, o1)
