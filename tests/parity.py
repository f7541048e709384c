"""Shared helpers of the GPU parity tests: run the CUDA path, run the oracle, compare.

Tolerances (fixed for the attention forward): on O, max |err| <= 2e-2 and
mean |err| <= 2e-3 over every compared element; on LSE,
|err| <= 1e-3 * max(1, |LSE_ref|).  Rows with no valid key must give O = 0
and LSE = -inf exactly.
"""
from __future__ import annotations

import numpy as np
import torch

import oracle
from paper_2609_18077_gb300 import binding, workloads

O_MAX_ABS = 2e-2
O_MEAN_ABS = 2e-3
LSE_REL = 1e-3


def gather_rows(t: torch.Tensor, rows):
    """[B,H,Sq,...] -> [B,H,n,...] at per-(b,h) row indices rows [B*H, n] (CPU numpy out)."""
    if rows is None:
        return t.cpu()
    B, H = t.shape[:2]
    idx = torch.from_numpy(rows.astype(np.int64)).to(t.device).view(B, H, -1)
    if t.dim() == 4:
        g = torch.gather(t, 2, idx.unsqueeze(-1).expand(-1, -1, -1, t.shape[3]))
    else:
        g = torch.gather(t, 2, idx)
    return g.cpu()


def compare(o_gpu, lse_gpu, o_ref, lse_ref, rows=None):
    """Assert the tolerances above; returns (max_abs, mean_abs, lse_rel_max)."""
    o = gather_rows(o_gpu, rows).float().double().numpy()
    assert o.shape == o_ref.shape
    assert np.all(np.isfinite(o)), "non-finite values in O"
    err = np.abs(o - o_ref)
    max_abs, mean_abs = float(err.max()), float(err.mean())
    assert max_abs <= O_MAX_ABS, f"O max abs err {max_abs}"
    assert mean_abs <= O_MEAN_ABS, f"O mean abs err {mean_abs}"
    lse_rel = 0.0
    if lse_gpu is not None:
        lse = gather_rows(lse_gpu, rows).double().numpy()
        empty = np.isneginf(lse_ref)
        assert np.array_equal(np.isneginf(lse), empty), "LSE -inf pattern differs"
        assert np.all(o[empty] == 0), "rows without keys must be zero"
        fin = ~empty
        if fin.any():
            rel = np.abs(lse[fin] - lse_ref[fin]) / np.maximum(1.0, np.abs(lse_ref[fin]))
            lse_rel = float(rel.max())
            assert lse_rel <= LSE_REL, f"LSE rel err {lse_rel}"
    return max_abs, mean_abs, lse_rel


def run_gpu(q, k, v, scale, kv_lens=None, device="cuda", with_lse=True, q_seg=None, kv_seg=None, window=None):
    """window: None or (grid, (kt, kh, kw), neighbourhood) for windowed 3D attention."""
    qd, kd, vd = (t.to(device) for t in (q, k, v))
    if window is not None:
        grid, ks, nb = window
        out, lse = binding.attn_fwd_win3d(qd, kd, vd, grid, ks, nb, scale=scale, return_lse=with_lse)
    elif q_seg is not None:
        qs = torch.from_numpy(np.ascontiguousarray(q_seg, dtype=np.int32)).to(device)
        ks = torch.from_numpy(np.ascontiguousarray(kv_seg, dtype=np.int32)).to(device)
        out, lse = binding.attn_fwd_segments(qd, kd, vd, qs, ks, scale=scale, return_lse=with_lse)
    elif kv_lens is None:
        out, lse = binding.attn_fwd(qd, kd, vd, scale=scale, return_lse=with_lse)
    else:
        lens = torch.from_numpy(np.asarray(kv_lens, dtype=np.int32)).to(device)
        out, lse = binding.attn_fwd_varlen(qd, kd, vd, lens, scale=scale, return_lse=with_lse)
    st = binding.check_device_error()
    assert st == binding.VDX_OK, binding.status_string(st)
    return out, lse


def run_oracle(q, k, v, scale, kv_lens=None, rows=None, q_seg=None, kv_seg=None, window=None):
    if window is not None:
        grid, ks, nb = window
        return oracle.attn_fwd_win3d(workloads.bf16_bits(q), workloads.bf16_bits(k), workloads.bf16_bits(v),
                                     scale, grid, ks, nb, rows=rows)
    return oracle.attn_fwd(workloads.bf16_bits(q), workloads.bf16_bits(k), workloads.bf16_bits(v),
                           scale, kv_lens=kv_lens, rows=rows, q_seg=q_seg, kv_seg=kv_seg)


def check_case(B, H, Sq, Skv, D, scale, seed, gain=1.0, kv_lens=None, rows=None, q_seg=None, kv_seg=None):
    q, k, v = workloads.random_qkv(B, H, Sq, Skv, D, seed, gain)
    if kv_lens is not None:
        k, v = workloads.pad_invalid_keys(k, v, kv_lens)
    out, lse = run_gpu(q, k, v, scale, kv_lens, q_seg=q_seg, kv_seg=kv_seg)
    o_ref, lse_ref = run_oracle(q, k, v, scale, kv_lens, rows, q_seg=q_seg, kv_seg=kv_seg)
    return compare(out, lse, o_ref, lse_ref, rows)
