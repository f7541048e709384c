"""Parity on the video-shaped workloads at full size, in the bench's launch
configuration, against the oracle on a seeded subset of query rows per head.

The subset is the workload's 4096 seeded query rows per (b, h), the sample
size the tolerances are stated for; VDX_PARITY_ROWS=n checks only the first
n of them (a quicker run while developing).
"""
import os

import numpy as np
import pytest
import torch

from parity import compare, run_gpu, run_oracle

pytestmark = pytest.mark.gpu

ROWS = int(os.environ.get("VDX_PARITY_ROWS", "4096"))


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_18077_gb300 import build, binding
    build.build()
    binding.load()


@pytest.mark.parametrize("name", ["tiny", "small480", "cross", "large480", "large720", "joint45k", "rope480",
                                  "win3d"])
def test_workload(name):
    from paper_2609_18077_gb300 import binding, workloads
    import oracle
    w = workloads.generate(name)
    rows = w["rows"]
    if rows is not None:
        rows = np.ascontiguousarray(rows[:, :ROWS])
    q, k = w["q"], w["k"]
    q_ref, k_ref = q, k
    wl = w["workload"]
    if wl.rope is not None:
        # GPU: rotate on the device, then attend; oracle: rotate in fp64, round to
        # bf16 (nearest even) as the model's tensors are, then attend in fp64
        grid, s0, dims, theta, inter = wl.rope
        q = binding.rope3d(q.cuda(), grid, s0, dims, theta, inter)
        k = binding.rope3d(k.cuda(), grid, s0, dims, theta, inter)
        q_ref = torch.from_numpy(oracle.rope3d(workloads.bf16_bits(w["q"]), grid, s0, dims, theta, inter)).to(
            torch.bfloat16)
        k_ref = torch.from_numpy(oracle.rope3d(workloads.bf16_bits(w["k"]), grid, s0, dims, theta, inter)).to(
            torch.bfloat16)
    window = None if wl.window is None else (wl.latent, wl.window[0], wl.window[1])
    out, lse = run_gpu(q, k, w["v"], w["scale"], w["kv_lens"], q_seg=w["q_seg"], kv_seg=w["kv_seg"],
                       window=window)
    o_ref, lse_ref = run_oracle(q_ref, k_ref, w["v"], w["scale"], w["kv_lens"], rows, q_seg=w["q_seg"],
                                kv_seg=w["kv_seg"], window=window)
    stats = compare(out, lse, o_ref, lse_ref, rows)
    print(f"{name}: O max {stats[0]:.3e} mean {stats[1]:.3e} LSE rel {stats[2]:.3e}")
    del out, lse
    torch.cuda.empty_cache()
