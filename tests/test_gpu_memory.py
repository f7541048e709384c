"""Device memory the library keeps: once a stream's split-tail scratch exists
(allocated at its bound by the first call that splits), later dense calls on
that stream allocate and free nothing, whatever their split; vdx_release
gives the stream's buffers back and the next call allocates again."""
import math

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


def _free():
    torch.cuda.synchronize()
    return torch.cuda.mem_get_info()[0]


def test_no_allocation_after_setup_and_release():
    from paper_2609_18077_gb300 import binding, workloads
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    D = 128
    # two heads and five heads more than multiprocessors: last rounds of 2
    # and 5 units, split into different numbers of parts
    cases = []
    for extra, seed in ((2, 31), (5, 32)):
        q, k, v = (t.cuda() for t in workloads.random_qkv(1, sms + extra, 256, 2000, D, seed=seed, logit_gain=1.3))
        cases.append((q, k, v, torch.empty_like(q), torch.empty(q.shape[:3], dtype=torch.float32, device="cuda")))
    first = [(torch.empty_like(o), torch.empty_like(l)) for *_, o, l in cases]   # copies of the first results
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        q, k, v, o, l = cases[0]
        binding.attn_fwd(q, k, v, scale=D ** -0.5, out=o, lse=l)          # set-up of this stream's scratch
        free0 = _free()
        for _ in range(3):
            for q, k, v, o, l in cases:
                binding.attn_fwd(q, k, v, scale=D ** -0.5, out=o, lse=l)
        free1 = _free()
        assert binding.check_device_error(torch.device("cuda", 0)) == binding.VDX_OK
        assert free1 == free0, f"dense calls after set-up changed free memory by {free0 - free1} bytes"
        for (*_, o, l), (o0, l0) in zip(cases, first):
            o0.copy_(o)
            l0.copy_(l)
        assert _free() == free1
        binding.release()
        free2 = _free()
        assert free2 > free1, "vdx_release freed nothing"
        for (q, k, v, o, l), (o0, l0) in zip(cases, first):
            binding.attn_fwd(q, k, v, scale=D ** -0.5, out=o, lse=l)       # allocates again
            torch.cuda.synchronize()
            assert torch.equal(o.view(torch.int16), o0.view(torch.int16)) and torch.equal(l, l0)
        binding.release()
    torch.cuda.current_stream().wait_stream(side)
    # the results themselves: the fp64 oracle on a few rows of the second case
    q, k, v, o, l = cases[1]
    rows = torch.arange(0, 256, 37, dtype=torch.int32).repeat(q.shape[1], 1).numpy()
    o_ref, l_ref = run_oracle(q.cpu(), k.cpu(), v.cpu(), 1 / math.sqrt(D), rows=rows)
    compare(o, l, o_ref, l_ref, rows)


def test_release_of_rope_and_host_buffers():
    """vdx_attn_fwd_rope3d keeps two turned copies of q and k and the host
    pipeline its slots; vdx_release frees both, and later calls still give
    the same results."""
    from paper_2609_18077_gb300 import binding, workloads
    B, H, S, D = 1, 4, 4 * 8 * 16, 128
    grid, dims = (4, 8, 16), (44, 42, 42)
    q, k, v = workloads.random_qkv(B, H, S, S, D, seed=41)
    qd, kd, vd = q.cuda(), k.cuda(), v.cuda()
    o1, l1 = binding.attn_fwd_rope3d(qd, kd, vd, grid, 0, dims, 1e4, True, scale=D ** -0.5)
    oh1, lh1 = binding.attn_fwd_host(q.pin_memory(), k.pin_memory(), v.pin_memory(), scale=D ** -0.5,
                                     device=torch.device("cuda", 0))
    free0 = _free()
    binding.release()
    free1 = _free()
    assert free1 > free0, "vdx_release freed nothing"
    o2, l2 = binding.attn_fwd_rope3d(qd, kd, vd, grid, 0, dims, 1e4, True, scale=D ** -0.5)
    oh2, lh2 = binding.attn_fwd_host(q.pin_memory(), k.pin_memory(), v.pin_memory(), scale=D ** -0.5,
                                     device=torch.device("cuda", 0))
    assert binding.check_device_error() == binding.VDX_OK
    assert torch.equal(o1.view(torch.int16), o2.view(torch.int16)) and torch.equal(l1, l2)
    assert torch.equal(oh1.view(torch.int16), oh2.view(torch.int16)) and torch.equal(lh1, lh2)
    binding.release()
