"""vdx_attn_fwd_host: attention forward on host buffers, copies overlapped
with the kernel.

Every chunk of the host path is one vdx_attn_fwd (or vdx_attn_fwd_varlen)
launch over a block of (b, h) rows, so the host path must give, bit for bit,
what device calls on the same blocks give -- and for varlen problems (no
key split) what one device call on the whole problem gives; it must also
match the oracle within the parity tolerances.
"""
import numpy as np
import pytest
import torch

from parity import compare, run_oracle

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_18077_gb300 import build, binding
    build.build()
    binding.load()


def _device_chunks(q, k, v, scale, r, with_lse=True):
    """vdx_attn_fwd over consecutive blocks of r flattened (b, h) rows."""
    from paper_2609_18077_gb300 import binding
    B, H, Sq, D = q.shape
    Skv = k.shape[2]
    qf, kf, vf = (t.cuda().view(B * H, -1, D) for t in (q, k, v))
    outs, lses = [], []
    for r0 in range(0, B * H, r):
        n = min(r, B * H - r0)
        o, l = binding.attn_fwd(qf[r0:r0 + n].unsqueeze(0), kf[r0:r0 + n].unsqueeze(0),
                                vf[r0:r0 + n].unsqueeze(0), scale=scale, return_lse=with_lse)
        outs.append(o[0].cpu())
        lses.append(None if l is None else l[0].cpu())
    out = torch.cat(outs).view(B, H, Sq, D)
    lse = None if not with_lse else torch.cat(lses).view(B, H, Sq)
    return out, lse


@pytest.mark.parametrize("B,H,Sq,Skv,D,r", [
    (1, 5, 300, 200, 128, 1),     # one row per chunk: five chunks through two slots
    (1, 5, 300, 200, 128, 2),     # ragged last chunk
    (1, 5, 300, 200, 128, 5),     # one chunk
    (2, 3, 513, 129, 64, 4),      # D = 64, chunk across the sample boundary
    (3, 4, 1100, 384, 128, 5),    # several query tile pairs per row
])
def test_dense_bit_identical_to_device_chunks(B, H, Sq, Skv, D, r):
    from paper_2609_18077_gb300 import binding, workloads
    q, k, v = workloads.random_qkv(B, H, Sq, Skv, D, 4100 + B * 100 + H * 10 + r, 2.0)
    scale = D ** -0.5
    out, lse = binding.attn_fwd_host(*(t.pin_memory() for t in (q, k, v)), scale=scale, chunk_rows=r)
    o_dev, l_dev = _device_chunks(q, k, v, scale, r)
    assert torch.equal(out, o_dev)
    assert torch.equal(lse, l_dev)
    o_ref, lse_ref = run_oracle(q, k, v, scale)
    compare(out, lse, o_ref, lse_ref)


def test_dense_auto_chunks_no_lse_pageable():
    """Library-chosen chunks, no LSE, pageable (not pinned) host buffers."""
    from paper_2609_18077_gb300 import binding, workloads
    q, k, v = workloads.random_qkv(2, 6, 700, 300, 128, 4201, 1.5)
    scale = 0.09
    out, lse = binding.attn_fwd_host(q, k, v, scale=scale, return_lse=False,
                                     out=torch.empty(q.shape, dtype=torch.bfloat16))
    assert lse is None
    o_ref, lse_ref = run_oracle(q, k, v, scale)
    compare(out, None, o_ref, lse_ref)


@pytest.mark.parametrize("r", [0, 1, 3, 4, 8, 12])
def test_varlen_bit_identical_to_one_device_call(r):
    """Chunks of heads of one sample (r <= H, ragged when H % r) or of whole
    samples (r = 8 rounds down to 4 = H, r = 12 is three samples)."""
    from paper_2609_18077_gb300 import binding, workloads
    B, H, Sq, Skv, D = 3, 4, 300, 256, 128
    lens = np.array([0, 1, 200], dtype=np.int32)
    q, k, v = workloads.random_qkv(B, H, Sq, Skv, D, 4300 + r, 2.0)
    k, v = workloads.pad_invalid_keys(k, v, lens)
    scale = D ** -0.5
    out, lse = binding.attn_fwd_host(*(t.pin_memory() for t in (q, k, v)), kv_lens=torch.from_numpy(lens),
                                     scale=scale, chunk_rows=r)
    o_dev, l_dev = binding.attn_fwd_varlen(q.cuda(), k.cuda(), v.cuda(), torch.from_numpy(lens).cuda(), scale=scale)
    assert torch.equal(out, o_dev.cpu())
    assert torch.equal(lse, l_dev.cpu())
    o_ref, lse_ref = run_oracle(q, k, v, scale, kv_lens=lens)
    compare(out, lse, o_ref, lse_ref)


def test_calls_are_stream_ordered():
    """A second call whose queries are the first call's output, enqueued
    before the first has finished, reads that output."""
    from paper_2609_18077_gb300 import binding, workloads
    q, k, v = (t.pin_memory() for t in workloads.random_qkv(1, 4, 600, 600, 128, 4401, 2.0))
    o1, _ = binding.attn_fwd_host(q, k, v, chunk_rows=1, synchronize=False)
    o2, l2 = binding.attn_fwd_host(o1, k, v, chunk_rows=1, synchronize=False)
    torch.cuda.current_stream().synchronize()
    r1, _ = binding.attn_fwd_host(q, k, v, chunk_rows=1)
    r2, s2 = binding.attn_fwd_host(r1, k, v, chunk_rows=1)
    assert torch.equal(o1, r1)
    assert torch.equal(o2, r2) and torch.equal(l2, s2)


@pytest.mark.parametrize("name", ["small480", "cross"])
def test_workload_host_path(name):
    """The bench's end-to-end path at full size: sampled rows against the
    oracle; the varlen workload also bit for bit against one device call."""
    from paper_2609_18077_gb300 import binding, workloads
    w = workloads.generate(name)
    rows = None if w["rows"] is None else np.ascontiguousarray(w["rows"][:, :256])
    q, k, v = (w[n].pin_memory() for n in ("q", "k", "v"))
    lens = None if w["kv_lens"] is None else torch.from_numpy(w["kv_lens"].astype(np.int32))
    out, lse = binding.attn_fwd_host(q, k, v, kv_lens=lens, scale=w["scale"])
    o_ref, lse_ref = run_oracle(w["q"], w["k"], w["v"], w["scale"], w["kv_lens"], rows)
    stats = compare(out, lse, o_ref, lse_ref, rows)
    print(f"{name} host path: O max {stats[0]:.3e} mean {stats[1]:.3e} LSE rel {stats[2]:.3e}")
    if lens is not None:
        o_dev, l_dev = binding.attn_fwd_varlen(w["q"].cuda(), w["k"].cuda(), w["v"].cuda(), lens.cuda(),
                                               scale=w["scale"])
        assert torch.equal(out, o_dev.cpu()) and torch.equal(lse, l_dev.cpu())
    torch.cuda.empty_cache()


@pytest.mark.parametrize("r", [0, 1, 2, 4, 6])
def test_segments_host_bit_identical_to_one_device_call(r):
    """Joint text-video ids (padded text slots in their own segment); chunks of
    heads of one sample (r <= H) or of whole samples (r = 4 rounds down to 3)."""
    from paper_2609_18077_gb300 import binding, workloads
    B, H, S, D = 2, 3, 700, 64
    seg = workloads.joint_segments([37, 120], 130, S)
    q, k, v = workloads.random_qkv(B, H, S, S, D, 4500 + r, 2.0)
    scale = D ** -0.5
    qs = torch.from_numpy(seg)
    out, lse = binding.attn_fwd_segments_host(*(t.pin_memory() for t in (q, k, v)), qs, qs, scale=scale,
                                              chunk_rows=r)
    o_dev, l_dev = binding.attn_fwd_segments(q.cuda(), k.cuda(), v.cuda(), qs.cuda(), qs.cuda(), scale=scale)
    assert torch.equal(out, o_dev.cpu())
    assert torch.equal(lse, l_dev.cpu())
    o_ref, lse_ref = run_oracle(q, k, v, scale, q_seg=seg, kv_seg=seg)
    compare(out, lse, o_ref, lse_ref)


@pytest.mark.parametrize("r", [0, 1, 5])
def test_win3d_host_bit_identical_to_one_device_call(r):
    from paper_2609_18077_gb300 import binding, workloads
    B, H, D = 1, 5, 128
    grid, window = (4, 6, 20), (3, 3, 5)
    S = grid[0] * grid[1] * grid[2]
    q, k, v = workloads.random_qkv(B, H, S, S, D, 4600 + r, 2.0)
    scale = D ** -0.5
    out, lse = binding.attn_fwd_win3d_host(*(t.pin_memory() for t in (q, k, v)), grid, window, True, scale=scale,
                                           chunk_rows=r)
    o_dev, l_dev = binding.attn_fwd_win3d(q.cuda(), k.cuda(), v.cuda(), grid, window, True, scale=scale)
    assert torch.equal(out, o_dev.cpu())
    assert torch.equal(lse, l_dev.cpu())
    o_ref, lse_ref = run_oracle(q, k, v, scale, window=(grid, window, True))
    compare(out, lse, o_ref, lse_ref)


@pytest.mark.parametrize("r", [0, 1, 3, 6])
def test_rope3d_host_bit_identical_to_device_chunks(r):
    """Each chunk turns its q and k rows in the device slot, then attends them:
    bit for bit vdx_rope3d on the whole tensors followed by vdx_attn_fwd on the
    same blocks of rows (one block: the device vdx_attn_fwd_rope3d call)."""
    from paper_2609_18077_gb300 import binding, workloads
    import oracle
    B, H, D = 2, 3, 128
    grid, s0, dims, theta = (3, 6, 10), 9, (44, 42, 42), 1e4
    S = s0 + grid[0] * grid[1] * grid[2] + 4
    q, k, v = workloads.random_qkv(B, H, S, S, D, 4700 + r, 1.5)
    scale = D ** -0.5
    out, lse = binding.attn_fwd_rope3d_host(*(t.pin_memory() for t in (q, k, v)), grid, s0, dims, theta, True,
                                            scale=scale, chunk_rows=r)
    qr = binding.rope3d(q.cuda(), grid, s0, dims, theta, True).cpu()
    kr = binding.rope3d(k.cuda(), grid, s0, dims, theta, True).cpu()
    if r == 0:
        o_dev, l_dev = binding.attn_fwd_rope3d(q.cuda(), k.cuda(), v.cuda(), grid, s0, dims, theta, True, scale=scale)
        o_dev, l_dev = o_dev.cpu(), l_dev.cpu()   # library-chosen chunks: compared to the oracle below
    else:
        o_dev, l_dev = _device_chunks(qr, kr, v, scale, r)
        assert torch.equal(out, o_dev)
        assert torch.equal(lse, l_dev)
    q_ref = torch.from_numpy(oracle.rope3d(workloads.bf16_bits(q), grid, s0, dims, theta, True)).to(torch.bfloat16)
    k_ref = torch.from_numpy(oracle.rope3d(workloads.bf16_bits(k), grid, s0, dims, theta, True)).to(torch.bfloat16)
    o_ref, lse_ref = run_oracle(q_ref, k_ref, v, scale)
    compare(out, lse, o_ref, lse_ref)
