"""Ulysses wrapper on one GPU: P ranks' exchange emulated in one process, each
rank's head-sharded attention run by the CUDA kernel one after another (no
kernel waits on another).  The gathered result is checked against the fp64
oracle over all heads at the parity tolerances, and bit for bit against one
CUDA call over all heads (Sec. 2 of the paper: the sequence-sharded
activations are exchanged into a head-sharded view for the attention op)."""
import math

import pytest
import torch

from parity import compare, run_oracle
from test_ulysses_cpu import _simulate

from paper_2609_18077_gb300 import binding, workloads

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_18077_gb300 import build
    build.build()
    binding.load()


@pytest.mark.parametrize("P", [2, 4])
def test_emulated_ranks_equal_one_call(P):
    # small enough that neither the full call nor a rank's call takes the split tail
    B, H, S, D = 1, 8, 1024, 128
    q, k, v = (t.cuda() for t in workloads.random_qkv(B, H, S, S, D, seed=62, logit_gain=1.5))
    scale = 1 / math.sqrt(D)
    s = S // P
    shards = [tuple(t[:, :, r * s:(r + 1) * s].contiguous() for t in (q, k, v)) for r in range(P)]
    outs, lses = _simulate(shards, lambda a, b, c: binding.attn_fwd(a, b, c, scale=scale))
    assert binding.check_device_error() == binding.VDX_OK
    o_seq, l_seq = torch.cat(outs, dim=2), torch.cat(lses, dim=2)
    # against the plain fp64 definition over all heads and the whole sequence
    o_ref, l_ref = run_oracle(q.cpu(), k.cpu(), v.cpu(), scale)
    compare(o_seq, l_seq, o_ref, l_ref)
    # and bit for bit against one kernel call over all heads
    o_full, l_full = binding.attn_fwd(q, k, v, scale=scale)
    assert binding.check_device_error() == binding.VDX_OK
    assert torch.equal(o_seq.view(torch.int16), o_full.view(torch.int16))
    assert torch.equal(l_seq, l_full)
