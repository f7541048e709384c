"""The C-ABI library loads, exports every declared symbol, and validates
arguments before any CUDA call (CPU only: no compute is launched)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "vdx.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2609_18077_gb300 import build, binding
    build.build()
    return binding.load()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(vdx_[a-z0-9_]+)\s*\(", text)))


def test_exports_every_declared_symbol(lib):
    from paper_2609_18077_gb300 import binding
    names = declared_functions()
    assert names, "no declarations found"
    for n in names:
        assert hasattr(lib, n), f"missing export {n}"
    assert sorted(binding.SIGNATURES) == names


def test_version_and_status(lib):
    from paper_2609_18077_gb300 import binding
    assert binding.version() == 10000
    for s in range(8):
        assert binding.status_string(s).startswith("VDX_")
    assert binding.status_string(99) == "unknown vdx status"


A = 0x10000  # fake, 16-byte aligned addresses: validation must reject before touching them
GOOD = dict(q=A, k=2 * A, v=3 * A, out=4 * A, lse=5 * A, B=1, H=1, Sq=8, Skv=8, D=128, scale=0.1)


def call(lib, **kw):
    a = {**GOOD, **kw}
    return lib.vdx_attn_fwd(a["q"], a["k"], a["v"], a["out"], a["lse"], a["B"], a["H"], a["Sq"], a["Skv"],
                            a["D"], a["scale"], None)


@pytest.mark.parametrize("kw,status", [
    (dict(q=None), 1), (dict(k=None), 1), (dict(v=None), 1), (dict(out=None), 1),
    (dict(D=96), 1), (dict(D=0), 1), (dict(B=-1), 1), (dict(Sq=-2), 1), (dict(Skv=-1), 1),
    (dict(scale=float("nan")), 1), (dict(scale=float("inf")), 1),
    (dict(q=A + 8), 3), (dict(out=4 * A + 2), 3), (dict(lse=5 * A + 2), 3),
    (dict(out=A), 1),                     # out overlaps q
    (dict(B=0), 0), (dict(Sq=0), 0), (dict(H=0), 0),   # empty: no-op, no CUDA call
])
def test_validation(lib, kw, status):
    assert call(lib, **kw) == status


@pytest.mark.parametrize("kw,status", [
    (dict(q=None), 1), (dict(out=None), 1), (dict(D=96), 1), (dict(B=-1), 1), (dict(scale=float("nan")), 1),
    (dict(q=A + 8), 3), (dict(out=4 * A + 2), 3), (dict(lse=5 * A + 2), 3),
    (dict(out=A), 1),                     # out overlaps q
    (dict(B=0), 0), (dict(Sq=0), 0),
])
def test_noalloc_validation_matches(lib, kw, status):
    """vdx_attn_fwd_noalloc rejects a bad call exactly as vdx_attn_fwd does,
    before any CUDA call (on this CPU-only machine a CUDA call would fail with
    VDX_ERR_CUDA instead)."""
    a = {**GOOD, **kw}
    args = (a["q"], a["k"], a["v"], a["out"], a["lse"], a["B"], a["H"], a["Sq"], a["Skv"], a["D"], a["scale"], None)
    assert lib.vdx_attn_fwd_noalloc(*args) == status
    assert lib.vdx_attn_fwd(*args) == status


def test_varlen_requires_lengths(lib):
    g = GOOD
    assert lib.vdx_attn_fwd_varlen(g["q"], g["k"], g["v"], g["out"], g["lse"], 1, 1, 8, 8, 128, None,
                                   0.1, None) == 1
    assert lib.vdx_attn_fwd_varlen(g["q"], g["k"], g["v"], g["out"], g["lse"], 1, 1, 8, 8, 128, 6 * A + 1,
                                   0.1, None) == 3


def test_segments_require_ids(lib):
    g = GOOD
    args = (g["q"], g["k"], g["v"], g["out"], g["lse"], 1, 1, 8, 8, 128)
    assert lib.vdx_attn_fwd_segments(*args, None, 7 * A, 0.1, None) == 1
    assert lib.vdx_attn_fwd_segments(*args, 6 * A, None, 0.1, None) == 1
    assert lib.vdx_attn_fwd_segments(*args, 6 * A + 2, 7 * A, 0.1, None) == 3
    assert lib.vdx_attn_fwd_segments(*args, 6 * A, 7 * A + 1, 0.1, None) == 3
    assert lib.vdx_attn_fwd_segments(g["q"], g["k"], g["v"], g["out"], g["lse"], 1, 1, 8, 8, 80,
                                     6 * A, 7 * A, 0.1, None) == 1
    assert lib.vdx_attn_fwd_segments(g["q"], g["k"], g["v"], g["out"], g["lse"], 0, 1, 8, 8, 128,
                                     6 * A, 7 * A, 0.1, None) == 0


@pytest.mark.parametrize("kw,status", [
    (dict(x=None), 1), (dict(y=None), 1), (dict(D=7), 1), (dict(D=0), 1), (dict(D=514), 1),
    (dict(d_t=3), 1), (dict(d_h=-2), 1), (dict(d_t=64, d_h=64, d_w=2), 1), (dict(theta=0.0), 1),
    (dict(theta=float("nan")), 1), (dict(B=-1), 1), (dict(F=-1), 1), (dict(s0=-1), 1),
    (dict(x=A + 2), 3), (dict(y=2 * A + 2), 3), (dict(y=A + 64), 1),   # overlapping, not equal
    (dict(B=0), 0), (dict(S=0), 0),
])
def test_rope_validation(lib, kw, status):
    a = dict(x=A, y=2 * A, B=1, H=1, S=8, D=128, F=2, Hp=2, Wp=2, s0=0, d_t=44, d_h=42, d_w=42, theta=1e4,
             interleaved=1)
    a.update(kw)
    assert lib.vdx_rope3d(a["x"], a["y"], a["B"], a["H"], a["S"], a["D"], a["F"], a["Hp"], a["Wp"], a["s0"],
                          a["d_t"], a["d_h"], a["d_w"], a["theta"], a["interleaved"], None) == status


def test_window_validation(lib):
    g = GOOD
    args = (g["q"], g["k"], g["v"], g["out"], g["lse"], 1, 1)
    assert lib.vdx_attn_fwd_win3d(*args, 2, 2, 2, 128, 4, 3, 3, 1, 0.1, None) == 1      # even window
    assert lib.vdx_attn_fwd_win3d(*args, 2, 2, 2, 128, 3, 0, 3, 1, 0.1, None) == 1      # empty window
    assert lib.vdx_attn_fwd_win3d(*args, -1, 2, 2, 128, 3, 3, 3, 1, 0.1, None) == 1
    assert lib.vdx_attn_fwd_win3d(*args, 2, 2, 2, 96, 3, 3, 3, 1, 0.1, None) == 1       # bad D
    assert lib.vdx_attn_fwd_win3d(*args, 70000, 70000, 2, 128, 3, 3, 3, 1, 0.1, None) == 2
    assert lib.vdx_attn_fwd_win3d(*args, 0, 2, 2, 128, 3, 3, 3, 1, 0.1, None) == 0       # no tokens


def test_selftest_limit_validation(lib):
    assert lib.vdx_selftest_wait_timeout(0, None) == 1
    assert lib.vdx_selftest_wait_timeout(10000001, None) == 1


def test_binding_rejects_cpu_tensors():
    import torch
    from paper_2609_18077_gb300 import binding
    x = torch.zeros(1, 1, 4, 64, dtype=torch.bfloat16)
    with pytest.raises(TypeError):
        binding.attn_fwd(x, x, x)


def test_host_entry_validation(lib):
    """vdx_attn_fwd_host rejects bad arguments before any CUDA call."""
    import torch
    q = torch.zeros(1, 2, 8, 64, dtype=torch.bfloat16)
    o = torch.zeros_like(q)
    lse = torch.zeros(1, 2, 8)
    a = (q.data_ptr(), q.data_ptr(), q.data_ptr())
    f = lib.vdx_attn_fwd_host
    assert f(None, *a[1:], o.data_ptr(), None, 1, 2, 8, 8, 64, None, 0.1, 0, None) == 1          # null q
    assert f(*a, None, None, 1, 2, 8, 8, 64, None, 0.1, 0, None) == 1                            # null out
    assert f(*a, o.data_ptr(), None, 1, 2, 8, 8, 96, None, 0.1, 0, None) == 1                    # bad D
    assert f(*a, o.data_ptr(), None, 1, -2, 8, 8, 64, None, 0.1, 0, None) == 1                   # negative H
    assert f(*a, o.data_ptr(), None, 1, 2, 8, 8, 64, None, 0.1, -1, None) == 1                   # chunk_rows < 0
    assert f(*a, o.data_ptr(), None, 1, 2, 8, 8, 64, None, float("nan"), 0, None) == 1           # scale
    assert f(*a, q.data_ptr(), None, 1, 2, 8, 8, 64, None, 0.1, 0, None) == 1                    # out aliases q
    assert f(*a, o.data_ptr(), ctypes.cast(o.data_ptr(), ctypes.c_void_p), 1, 2, 8, 8, 64, None, 0.1, 0,
             None) == 1                                                                          # lse inside out
    assert f(*a, o.data_ptr(), lse.data_ptr(), 0, 2, 8, 8, 64, None, 0.1, 0, None) == 0          # no rows
    assert f(*a, o.data_ptr(), lse.data_ptr(), 1, 2, 0, 8, 64, None, 0.1, 0, None) == 0          # no queries


def test_binding_host_entry_rejects_cuda_layouts():
    import torch
    from paper_2609_18077_gb300 import binding
    x = torch.zeros(1, 1, 4, 64, dtype=torch.float32)
    with pytest.raises(TypeError):
        binding.attn_fwd_host(x, x, x)
    y = torch.zeros(1, 1, 4, 64, dtype=torch.bfloat16)
    with pytest.raises(TypeError):
        binding.attn_fwd_host(y, y, y, kv_lens=torch.zeros(2, dtype=torch.int32))


def test_segment_and_window_host_entries_validate(lib):
    """The segment and window host entries reject bad arguments before any CUDA call."""
    import torch
    q = torch.zeros(1, 2, 8, 64, dtype=torch.bfloat16)
    o = torch.zeros_like(q)
    ids = torch.zeros(1, 8, dtype=torch.int32)
    a = (q.data_ptr(), q.data_ptr(), q.data_ptr(), o.data_ptr(), None)
    f = lib.vdx_attn_fwd_segments_host
    assert f(*a, 1, 2, 8, 8, 64, None, ids.data_ptr(), 0.1, 0, None) == 1                  # no q_seg
    assert f(*a, 1, 2, 8, 8, 64, ids.data_ptr(), None, 0.1, 0, None) == 1                  # no kv_seg
    assert f(*a, 1, 2, 8, 8, 64, ids.data_ptr(), ids.data_ptr(), 0.1, -3, None) == 1       # chunk_rows
    assert f(*a, 0, 2, 8, 8, 64, ids.data_ptr(), ids.data_ptr(), 0.1, 0, None) == 0        # no rows
    g = lib.vdx_attn_fwd_win3d_host
    assert g(*a, 1, 2, 2, 2, 2, 64, 2, 3, 3, 1, 0.1, 0, None) == 1                        # even window
    assert g(*a, 1, 2, 70000, 1, 1, 64, 3, 3, 3, 1, 0.1, 0, None) == 2                    # grid side
    assert g(*a, 1, 2, 2, 2, 2, 96, 3, 3, 3, 1, 0.1, 0, None) == 1                        # bad D
    assert g(*a, 1, 2, 0, 2, 2, 64, 3, 3, 3, 1, 0.1, 0, None) == 0                        # no tokens
    from paper_2609_18077_gb300 import binding
    with pytest.raises(TypeError):
        binding.attn_fwd_segments_host(q, q, q, ids, torch.zeros(1, 7, dtype=torch.int32))


def test_rope_attention_validates(lib):
    """vdx_attn_fwd_rope3d rejects bad arguments before any CUDA call."""
    g = GOOD
    f = lib.vdx_attn_fwd_rope3d
    base = dict(B=1, H=1, S=8, D=128, F=2, Hp=2, Wp=2, s0=0, dt=44, dh=42, dw=42, theta=1e4, inter=1, scale=0.1)

    def call(**kw):
        a = {**base, **kw}
        return f(g["q"], g["k"], g["v"], g["out"], g["lse"], a["B"], a["H"], a["S"], a["D"], a["F"], a["Hp"],
                 a["Wp"], a["s0"], a["dt"], a["dh"], a["dw"], a["theta"], a["inter"], a["scale"], None)
    assert call(D=96, dt=32, dh=32, dw=32) == 1       # attention needs D 64 or 128
    assert call(dt=45) == 1                            # odd part
    assert call(dt=64, dh=64, dw=8) == 1               # parts wider than D
    assert call(theta=-1.0) == 1
    assert call(scale=float("nan")) == 1
    assert call(B=-1) == 1
    assert call(S=0) == 0                              # nothing to do
    assert f(g["q"] + 8, g["k"], g["v"], g["out"], g["lse"], 1, 1, 8, 128, 2, 2, 2, 0, 44, 42, 42, 1e4, 1, 0.1,
             None) == 3                                # q not 16-byte aligned


def test_rope3d_host_validates(lib):
    import torch
    q = torch.zeros(1, 1, 8, 128, dtype=torch.bfloat16)
    o = torch.zeros_like(q)
    f = lib.vdx_attn_fwd_rope3d_host
    a = (q.data_ptr(), q.data_ptr(), q.data_ptr(), o.data_ptr(), None, 1, 1, 8, 128)
    assert f(*a, 2, 2, 2, 0, 45, 42, 42, 1e4, 1, 0.1, 0, None) == 1     # odd part
    assert f(*a, 2, 2, 2, 0, 44, 42, 42, 0.0, 1, 0.1, 0, None) == 1     # theta
    assert f(*a, 2, 2, 2, -1, 44, 42, 42, 1e4, 1, 0.1, 0, None) == 1    # s0
    assert f(*a, 2, 2, 2, 0, 44, 42, 42, 1e4, 1, 0.1, -1, None) == 1    # chunk_rows
