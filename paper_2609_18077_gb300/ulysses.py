"""Head-sharded (Ulysses) sequence-parallel attention over torch.distributed.

The vidax paper (Sec. 2, "Spatiotemporal tensor and sequence sharding")
shards temporal tokens across devices and, for the attention op only,
switches to a head-sharded view with all_to_all transposes (DeepSpeed-
Ulysses).  With P ranks, rank r holds the sequence shard
[r*S/P, (r+1)*S/P) of every head:

    q, k, v on rank r : [B, H, S/P, D]
    all_to_all        : rank r receives heads [r*H/P, (r+1)*H/P) of every shard
    local attention   : [B, H/P, S, D] (the whole sequence of its heads)
    all_to_all        : O and LSE go back to the sequence shards
    out, lse on rank r: [B, H, S/P, D], [B, H, S/P]

The local attention is the library's (vdx_attn_fwd, or
vdx_attn_fwd_segments with each sample's full-length segment ids); the
wrapper only moves data.  H and S must be multiples of P.  The pack and
unpack steps are plain functions, so that a test can run the exchange of P
ranks inside one process.
"""
from __future__ import annotations

import torch
import torch.distributed as dist


def pack_seq_to_head(x: torch.Tensor, P: int) -> torch.Tensor:
    """[B, H, s, ...] -> [P, B, H/P, s, ...]: chunk p holds head group p (sent to rank p)."""
    B, H = x.shape[:2]
    if H % P:
        raise ValueError(f"{H} heads do not split over {P} ranks")
    rest = x.shape[2:]
    return x.reshape(B, P, H // P, *rest).movedim(1, 0).contiguous()


def unpack_seq_to_head(recv: torch.Tensor) -> torch.Tensor:
    """[P, B, h, s, ...] (chunk p = sequence shard p) -> [B, h, P*s, ...]."""
    P, B, h, s = recv.shape[:4]
    rest = recv.shape[4:]
    return recv.movedim(0, 2).reshape(B, h, P * s, *rest).contiguous()


def pack_head_to_seq(y: torch.Tensor, P: int) -> torch.Tensor:
    """[B, h, S, ...] -> [P, B, h, S/P, ...]: chunk p holds sequence shard p (sent to rank p)."""
    B, h, S = y.shape[:3]
    if S % P:
        raise ValueError(f"{S} tokens do not split over {P} ranks")
    rest = y.shape[3:]
    return y.reshape(B, h, P, S // P, *rest).movedim(2, 0).contiguous()


def unpack_head_to_seq(recv: torch.Tensor) -> torch.Tensor:
    """[P, B, h, s, ...] (chunk p = head group p) -> [B, P*h, s, ...]."""
    P, B, h, s = recv.shape[:4]
    rest = recv.shape[4:]
    return recv.movedim(0, 1).reshape(B, P * h, s, *rest).contiguous()


def _exchange(send: torch.Tensor, group=None) -> torch.Tensor:
    recv = torch.empty_like(send)
    dist.all_to_all_single(recv, send, group=group)
    return recv


def ulysses_attention(q, k, v, scale=None, q_seg=None, kv_seg=None, group=None, local_attn=None):
    """Sequence-sharded attention through a head-sharded local call.

    q, k, v: this rank's sequence shard [B, H, S/P, D] (same shard size on
    every rank).  q_seg / kv_seg: optional int32 [B, S] segment ids of the
    whole sequence (the same on every rank).  local_attn(q, k, v, scale,
    q_seg, kv_seg) -> (out, lse) runs the head-sharded attention; by default
    the library's kernels.  Returns (out [B, H, S/P, D], lse [B, H, S/P]).
    """
    P = dist.get_world_size(group)
    if local_attn is None:
        local_attn = _library_attention
    qh, kh, vh = (unpack_seq_to_head(_exchange(pack_seq_to_head(t, P), group)) for t in (q, k, v))
    out, lse = local_attn(qh, kh, vh, scale, q_seg, kv_seg)
    out = unpack_head_to_seq(_exchange(pack_head_to_seq(out, P), group))
    lse = unpack_head_to_seq(_exchange(pack_head_to_seq(lse, P), group))
    return out, lse


def _library_attention(q, k, v, scale, q_seg, kv_seg):
    from . import binding
    if q_seg is not None:
        return binding.attn_fwd_segments(q, k, v, q_seg, kv_seg, scale=scale)
    return binding.attn_fwd(q, k, v, scale=scale)
