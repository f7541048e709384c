"""Ulysses head-sharded wrapper on CPU ranks (gloo) and in-process layout checks.

The wrapper only moves data: sequence shards -> all_to_all -> head groups over
the whole sequence -> local attention -> all_to_all back.  With the fp64
oracle as the local attention (test infrastructure), the gathered result must
equal one oracle call on the whole tensors exactly.
"""
import os
import socket

import numpy as np
import pytest
import torch
import torch.multiprocessing as mp

from paper_2609_18077_gb300 import ulysses, workloads


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _simulate(shards, local):
    """Run the wrapper's exchange for P in-process ranks; local(q, k, v) -> (out, lse)."""
    P = len(shards)
    send = [[ulysses.pack_seq_to_head(t, P) for t in sh] for sh in shards]
    heads = [[ulysses.unpack_seq_to_head(torch.stack([send[p][i][r] for p in range(P)])) for i in range(3)]
             for r in range(P)]
    res = [local(*h) for h in heads]
    back_o = [ulysses.pack_head_to_seq(o, P) for o, _ in res]
    back_l = [ulysses.pack_head_to_seq(l, P) for _, l in res]
    outs = [ulysses.unpack_head_to_seq(torch.stack([back_o[p][r] for p in range(P)])) for r in range(P)]
    lses = [ulysses.unpack_head_to_seq(torch.stack([back_l[p][r] for p in range(P)])) for r in range(P)]
    return outs, lses


@pytest.mark.parametrize("P", [1, 2, 4])
def test_layout_round_trip(P):
    """An identity 'attention' returns every rank its own shard: the two
    exchanges are inverse and keep the token order."""
    B, H, S, D = 2, 8, 16, 4
    x = torch.arange(B * H * S * D, dtype=torch.float64).view(B, H, S, D)
    s = S // P
    shards = [(x[:, :, r * s:(r + 1) * s],) * 3 for r in range(P)]

    def ident(q, k, v):
        assert q.shape == (B, H // P, S, D)
        return q, q[..., 0]

    outs, lses = _simulate(shards, ident)
    for r in range(P):
        assert torch.equal(outs[r], x[:, :, r * s:(r + 1) * s])
        assert torch.equal(lses[r], x[:, :, r * s:(r + 1) * s, 0])


def test_rejects_indivisible_heads():
    with pytest.raises(ValueError):
        ulysses.pack_seq_to_head(torch.zeros(1, 6, 4, 2), 4)
    with pytest.raises(ValueError):
        ulysses.pack_head_to_seq(torch.zeros(1, 2, 6, 2), 4)


def _oracle_local(q, k, v, scale, q_seg, kv_seg):
    import oracle
    o, lse = oracle.attn_fwd(workloads.bf16_bits(q), workloads.bf16_bits(k), workloads.bf16_bits(v), scale,
                             q_seg=None if q_seg is None else q_seg.numpy(),
                             kv_seg=None if kv_seg is None else kv_seg.numpy())
    return torch.from_numpy(o), torch.from_numpy(lse)


def _rank(rank, world, port, segments, q, k, v, seg, result):
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    s = q.shape[2] // world
    sl = slice(rank * s, (rank + 1) * s)
    q_seg = kv_seg = torch.from_numpy(seg) if segments else None
    out, lse = ulysses.ulysses_attention(q[:, :, sl].contiguous(), k[:, :, sl].contiguous(), v[:, :, sl].contiguous(),
                                         0.25, q_seg, kv_seg, local_attn=_oracle_local)
    result[rank] = (out, lse)
    dist.destroy_process_group()


@pytest.mark.parametrize("world,segments", [(2, False), (4, False), (2, True)])
def test_gloo_ranks_equal_one_call(world, segments):
    import oracle
    B, H, S, D = 2, 4, 48, 16
    q, k, v = workloads.random_qkv(B, H, S, S, D, seed=61, logit_gain=1.3)
    seg = workloads.joint_segments(np.array([5, 12], np.int32), 16, S)
    mgr = mp.get_context("spawn").Manager()
    result = mgr.dict()
    mp.spawn(_rank, args=(world, _free_port(), segments, q, k, v, seg, result), nprocs=world, join=True)
    kw = dict(q_seg=seg, kv_seg=seg) if segments else {}
    o_ref, lse_ref = oracle.attn_fwd(workloads.bf16_bits(q), workloads.bf16_bits(k), workloads.bf16_bits(v), 0.25,
                                     **kw)
    out = torch.cat([result[r][0] for r in range(world)], dim=2).numpy()
    lse = torch.cat([result[r][1] for r in range(world)], dim=2).numpy()
    np.testing.assert_array_equal(out, o_ref)
    np.testing.assert_array_equal(lse, lse_ref)
