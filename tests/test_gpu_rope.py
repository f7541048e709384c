"""3D rotary position embedding: CUDA path vs the fp64 oracle (GB300 only).

Tolerance from the arithmetic: the output is bf16 rounded to nearest, at most
half an ulp = 2^-8 |y| off the exact value, plus the fp32 sine, cosine and
product error, bounded by 2e-5 of the row's largest |x|.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_18077_gb300 import binding, workloads

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_18077_gb300 import build
    build.build()
    binding.load()


def _check(y_gpu, x, y_ref):
    y = y_gpu.float().double().cpu().numpy()
    xd = x.float().double().numpy()
    bound = 2.0 ** -8 * np.abs(y_ref) + 2e-5 * np.max(np.abs(xd), axis=-1, keepdims=True)
    err = np.abs(y - y_ref)
    assert np.all(np.isfinite(y))
    assert np.all(err <= bound), f"max excess {np.max(err - bound)} at {np.unravel_index(np.argmax(err - bound), err.shape)}"
    return float(err.max())


CASES = [
    # B, H, D, grid (F, Hp, Wp), s0, tokens after the grid, dims, theta, interleaved
    (1, 2, 128, (3, 4, 5), 0, 0, (44, 42, 42), 1e4, True),
    (2, 3, 128, (3, 4, 5), 7, 5, (44, 42, 42), 1e4, True),
    (2, 3, 128, (3, 4, 5), 7, 5, (16, 56, 56), 256.0, False),
    (1, 2, 64, (5, 3, 7), 3, 0, (16, 24, 20), 1e4, False),
    (1, 1, 64, (2, 6, 6), 0, 1, (8, 8, 8), 500.0, True),      # dims past the rotated parts copied
    (3, 1, 96, (1, 1, 33), 2, 2, (0, 0, 96), 10.0, True),    # one axis only
]


@pytest.mark.parametrize("B,H,D,grid,s0,after,dims,theta,inter", CASES)
@pytest.mark.parametrize("in_place", [False, True])
def test_rope_cases(B, H, D, grid, s0, after, dims, theta, inter, in_place):
    S = s0 + grid[0] * grid[1] * grid[2] + after
    x, _, _ = workloads.random_qkv(B, H, S, 1, D, seed=700 + S + D, logit_gain=1.5)
    y_ref = oracle.rope3d(workloads.bf16_bits(x), grid, s0, dims, theta, inter)
    xd = x.cuda()
    if in_place:
        y = binding.rope3d(xd, grid, s0, dims, theta, inter, out=xd)
        assert y.data_ptr() == xd.data_ptr()
    else:
        y = binding.rope3d(xd, grid, s0, dims, theta, inter)
        assert torch.equal(xd.cpu().view(torch.int16), x.view(torch.int16))   # input untouched
    assert binding.check_device_error() == binding.VDX_OK
    _check(y, x, y_ref)


def test_rope_small480_rows():
    """The small-DiT 480p geometry (21x30x52 grid, Wan's 44/42/42 split) at full
    size, checked on two whole (b, h) rows."""
    w = workloads.generate("small480")
    grid, dims = (21, 30, 52), (44, 42, 42)
    q = w["q"]
    y = binding.rope3d(q.cuda(), grid, 0, dims, 1e4, True)
    assert binding.check_device_error() == binding.VDX_OK
    for h in (0, 11):
        xs = q[:, h:h + 1].contiguous()
        y_ref = oracle.rope3d(workloads.bf16_bits(xs), grid, 0, dims, 1e4, True)
        _check(y[:, h:h + 1], xs, y_ref)


def test_rope_not_16_byte_aligned():
    """A tensor 4 bytes off a 16-byte boundary takes the per-pair kernel; same result."""
    B, H, D, grid, s0 = 1, 2, 128, (2, 3, 4), 1
    S = s0 + 24
    x, _, _ = workloads.random_qkv(B, H, S, 1, D, seed=801)
    y_ref = oracle.rope3d(workloads.bf16_bits(x), grid, s0, (44, 42, 42), 1e4, True)
    buf = torch.empty(x.numel() + 2, dtype=torch.bfloat16, device="cuda")
    xs = buf[2:].view(x.shape)
    xs.copy_(x.cuda())
    assert xs.data_ptr() % 16 == 4
    y = binding.rope3d(xs, grid, s0, (44, 42, 42), 1e4, True)
    assert binding.check_device_error() == binding.VDX_OK
    _check(y, x, y_ref)


# RoPE + attention in one call: B, H, D, grid, s0, tokens after the grid, dims, theta, interleaved
ROPE_ATTN = [
    (1, 3, 128, (3, 5, 7), 0, 0, (44, 42, 42), 1e4, True),       # S = 105: one ragged query tile pair
    (2, 2, 128, (4, 6, 11), 20, 13, (44, 42, 42), 1e4, True),    # text before, tokens after the grid
    (1, 2, 64, (5, 8, 9), 7, 0, (24, 20, 20), 1e4, True),         # D = 64 (two Q buffers)
    (1, 2, 128, (2, 9, 20), 0, 5, (16, 16, 16), 300.0, True),     # dims past the rotated parts unturned
    (1, 2, 128, (3, 5, 7), 3, 2, (44, 42, 42), 1e4, False),      # half-split pairs
    (1, 1, 128, (8, 16, 16), 0, 0, (44, 42, 42), 1e4, True),      # 2048 tokens: several units per CTA
]


@pytest.mark.parametrize("B,H,D,grid,s0,after,dims,theta,inter", ROPE_ATTN)
def test_rope_attention_bit_identical_to_separate_calls(B, H, D, grid, s0, after, dims, theta, inter):
    """vdx_attn_fwd_rope3d gives, bit for bit, vdx_rope3d on q and k followed
    by vdx_attn_fwd, leaves q and k untouched, and matches the oracle."""
    import oracle
    S = s0 + grid[0] * grid[1] * grid[2] + after
    q, k, v = workloads.random_qkv(B, H, S, S, D, seed=800 + S + D, logit_gain=1.5)
    qd, kd, vd = q.cuda(), k.cuda(), v.cuda()
    scale = D ** -0.5
    out, lse = binding.attn_fwd_rope3d(qd, kd, vd, grid, s0, dims, theta, inter, scale=scale)
    assert binding.check_device_error() == binding.VDX_OK
    assert torch.equal(qd.cpu().view(torch.int16), q.view(torch.int16))
    assert torch.equal(kd.cpu().view(torch.int16), k.view(torch.int16))
    qr = binding.rope3d(qd, grid, s0, dims, theta, inter)
    kr = binding.rope3d(kd, grid, s0, dims, theta, inter)
    o_sep, l_sep = binding.attn_fwd(qr, kr, vd, scale=scale)
    assert torch.equal(out, o_sep)
    assert torch.equal(lse, l_sep)
    from parity import compare
    q_ref = torch.from_numpy(oracle.rope3d(workloads.bf16_bits(q), grid, s0, dims, theta, inter)).to(torch.bfloat16)
    k_ref = torch.from_numpy(oracle.rope3d(workloads.bf16_bits(k), grid, s0, dims, theta, inter)).to(torch.bfloat16)
    o_ref, lse_ref = oracle.attn_fwd(workloads.bf16_bits(q_ref), workloads.bf16_bits(k_ref), workloads.bf16_bits(v),
                                     scale)
    compare(out, lse, o_ref, lse_ref)


def test_rope_attention_rope480():
    """The rope480 workload through the one call: bit for bit the separate
    calls, and the oracle on a seeded row sample."""
    import oracle
    from parity import compare
    w = workloads.generate("rope480")
    grid, s0, dims, theta, inter = w["workload"].rope
    qd, kd, vd = (w[n].cuda() for n in ("q", "k", "v"))
    out, lse = binding.attn_fwd_rope3d(qd, kd, vd, grid, s0, dims, theta, inter, scale=w["scale"])
    o_sep, l_sep = binding.attn_fwd(binding.rope3d(qd, grid, s0, dims, theta, inter),
                                    binding.rope3d(kd, grid, s0, dims, theta, inter), vd, scale=w["scale"])
    assert torch.equal(out, o_sep) and torch.equal(lse, l_sep)
    rows = np.ascontiguousarray(w["rows"][:, :256])
    q_ref = torch.from_numpy(oracle.rope3d(workloads.bf16_bits(w["q"]), grid, s0, dims, theta, inter)).to(torch.bfloat16)
    k_ref = torch.from_numpy(oracle.rope3d(workloads.bf16_bits(w["k"]), grid, s0, dims, theta, inter)).to(torch.bfloat16)
    o_ref, lse_ref = oracle.attn_fwd(workloads.bf16_bits(q_ref), workloads.bf16_bits(k_ref), workloads.bf16_bits(w["v"]),
                                     w["scale"], rows=rows)
    compare(out, lse, o_ref, lse_ref, rows)
    del out, lse, o_sep, l_sep
    torch.cuda.empty_cache()
