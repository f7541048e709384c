"""ctypes binding of libvdx (include/vdx.h): argument marshalling only.

Every step of the attention forward runs in the CUDA library; this module
checks tensor metadata, allocates outputs through PyTorch when the caller
does not pass them, and forwards raw device pointers, sizes and the current
CUDA stream.  There is no fallback: if the library is missing or the call
fails, an exception is raised.
"""
from __future__ import annotations

import ctypes
import math
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_lib", "libvdx.so")

VDX_OK = 0
VDX_ERR_INVALID_ARG = 1
VDX_ERR_UNSUPPORTED = 2
VDX_ERR_MISALIGNED = 3
VDX_ERR_CUDA = 4
VDX_ERR_DEVICE = 5
VDX_ERR_TIMEOUT = 6
VDX_ERR_DRAIN = 7

# Every symbol include/vdx.h declares, with its ctypes signature.
_P = ctypes.c_void_p
_I = ctypes.c_int
SIGNATURES = {
    "vdx_attn_fwd": (_I, [_P, _P, _P, _P, _P, _I, _I, _I, _I, _I, ctypes.c_float, _P]),
    "vdx_attn_fwd_varlen": (_I, [_P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _P, ctypes.c_float, _P]),
    "vdx_attn_fwd_segments": (_I, [_P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _P, _P, ctypes.c_float, _P]),
    "vdx_attn_fwd_noalloc": (_I, [_P, _P, _P, _P, _P, _I, _I, _I, _I, _I, ctypes.c_float, _P]),
    "vdx_attn_fwd_win3d": (_I, [_P, _P, _P, _P, _P] + [_I] * 10 + [ctypes.c_float, _P]),
    "vdx_rope3d": (_I, [_P, _P, _I, _I, _I, _I, _I, _I, _I, _I, _I, _I, _I, ctypes.c_float, _I, _P]),
    "vdx_attn_fwd_rope3d": (_I, [_P, _P, _P, _P, _P] + [_I] * 11 + [ctypes.c_float, _I, ctypes.c_float, _P]),
    "vdx_attn_fwd_host": (_I, [_P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _P, ctypes.c_float, ctypes.c_longlong, _P]),
    "vdx_attn_fwd_segments_host": (_I, [_P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _P, _P, ctypes.c_float,
                                        ctypes.c_longlong, _P]),
    "vdx_attn_fwd_win3d_host": (_I, [_P, _P, _P, _P, _P] + [_I] * 10 + [ctypes.c_float, ctypes.c_longlong, _P]),
    "vdx_attn_fwd_rope3d_host": (_I, [_P, _P, _P, _P, _P] + [_I] * 11 + [ctypes.c_float, _I, ctypes.c_float,
                                                                         ctypes.c_longlong, _P]),
    "vdx_status_string": (ctypes.c_char_p, [_I]),
    "vdx_check_device_error": (_I, [_P]),
    "vdx_release": (_I, [_P]),
    "vdx_selftest_wait_timeout": (_I, [_I, _P]),
    "vdx_version": (_I, []),
}

_lib = None


class VdxError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} (status {status})")


def load() -> ctypes.CDLL:
    """Load libvdx.so (built in-tree by ``__graft_entry__.build()``)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(
                f"CUDA library {LIB_PATH} is not built; run `python -c \"import __graft_entry__ as g; g.build()\"`")
        lib = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
    return _lib


def status_string(status: int) -> str:
    return load().vdx_status_string(int(status)).decode()


def version() -> int:
    return int(load().vdx_version())


def _stream_handle(device: torch.device):
    return ctypes.c_void_p(torch.cuda.current_stream(device).cuda_stream)


def check_device_error(device=None) -> int:
    """Synchronise the current stream and read/clear the device error word."""
    device = torch.device("cuda", torch.cuda.current_device()) if device is None else torch.device(device)
    with torch.cuda.device(device):
        return int(load().vdx_check_device_error(_stream_handle(device)))


def release(device=None) -> None:
    """Free the device memory the library keeps for the current stream of `device`."""
    device = torch.device("cuda", torch.cuda.current_device()) if device is None else torch.device(device)
    with torch.cuda.device(device):
        st = int(load().vdx_release(_stream_handle(device)))
    if st != VDX_OK:
        raise VdxError(st, "vdx_release")


def selftest_wait_timeout(limit_us: int, device=None) -> int:
    """Launch the bounded-wait self-test kernel; returns the launch status."""
    device = torch.device("cuda", torch.cuda.current_device()) if device is None else torch.device(device)
    with torch.cuda.device(device):
        return int(load().vdx_selftest_wait_timeout(int(limit_us), _stream_handle(device)))


def _check_qkv(q, k, v):
    for name, t in (("q", q), ("k", k), ("v", v)):
        if not isinstance(t, torch.Tensor) or not t.is_cuda:
            raise TypeError(f"{name} must be a CUDA tensor")
        if t.dtype != torch.bfloat16 or t.dim() != 4 or not t.is_contiguous():
            raise TypeError(f"{name} must be a contiguous bf16 [B,H,S,D] tensor")
    if k.shape != v.shape or q.shape[:2] != k.shape[:2] or q.shape[3] != k.shape[3]:
        raise ValueError(f"shape mismatch q{tuple(q.shape)} k{tuple(k.shape)} v{tuple(v.shape)}")
    if not (q.device == k.device == v.device):
        raise ValueError("q, k, v must be on one device")


def _outputs(q, out, lse, return_lse):
    B, H, Sq, D = q.shape
    if out is None:
        out = torch.empty_like(q)
    elif out.shape != q.shape or out.dtype != torch.bfloat16 or not out.is_contiguous() or out.device != q.device:
        raise ValueError("out must be a contiguous bf16 tensor shaped like q on q's device")
    if lse is None and return_lse:
        lse = torch.empty((B, H, Sq), dtype=torch.float32, device=q.device)
    elif lse is not None and (lse.shape != (B, H, Sq) or lse.dtype != torch.float32 or not lse.is_contiguous()
                              or lse.device != q.device):
        raise ValueError("lse must be a contiguous fp32 [B,H,Sq] tensor on q's device")
    return out, lse


def attn_fwd(q, k, v, scale=None, out=None, lse=None, return_lse=True):
    """Softmax attention forward through ``vdx_attn_fwd``.

    q: bf16 [B,H,Sq,D]; k, v: bf16 [B,H,Skv,D] (CUDA, contiguous).
    scale defaults to 1/sqrt(D).  Returns (out bf16 [B,H,Sq,D], lse fp32 [B,H,Sq] or None).
    """
    _check_qkv(q, k, v)
    B, H, Sq, D = q.shape
    Skv = k.shape[2]
    scale = 1.0 / math.sqrt(D) if scale is None else float(scale)
    out, lse = _outputs(q, out, lse, return_lse)
    with torch.cuda.device(q.device):
        st = load().vdx_attn_fwd(q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(),
                                 lse.data_ptr() if lse is not None else None,
                                 B, H, Sq, Skv, D, scale, _stream_handle(q.device))
    if st != VDX_OK:
        raise VdxError(st, "vdx_attn_fwd")
    return out, lse


def attn_fwd_varlen(q, k, v, kv_lens, scale=None, out=None, lse=None, return_lse=True):
    """Cross-attention to padded keys through ``vdx_attn_fwd_varlen``.

    kv_lens: int32 CUDA tensor [B] of valid key counts (keys past it are ignored).
    """
    _check_qkv(q, k, v)
    B, H, Sq, D = q.shape
    Skv_max = k.shape[2]
    if (not isinstance(kv_lens, torch.Tensor) or kv_lens.dtype != torch.int32 or kv_lens.shape != (B,)
            or kv_lens.device != q.device or not kv_lens.is_contiguous()):
        raise TypeError("kv_lens must be a contiguous int32 CUDA tensor of shape [B] on q's device")
    scale = 1.0 / math.sqrt(D) if scale is None else float(scale)
    out, lse = _outputs(q, out, lse, return_lse)
    with torch.cuda.device(q.device):
        st = load().vdx_attn_fwd_varlen(q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(),
                                        lse.data_ptr() if lse is not None else None,
                                        B, H, Sq, Skv_max, D, kv_lens.data_ptr(), scale,
                                        _stream_handle(q.device))
    if st != VDX_OK:
        raise VdxError(st, "vdx_attn_fwd_varlen")
    return out, lse


def attn_fwd_segments(q, k, v, q_seg, kv_seg, scale=None, out=None, lse=None, return_lse=True):
    """Joint attention with segment ids through ``vdx_attn_fwd_segments``.

    q_seg: int32 CUDA tensor [B, Sq]; kv_seg: int32 CUDA tensor [B, Skv]; query i
    of sample b attends the keys j with kv_seg[b, j] == q_seg[b, i].
    """
    _check_qkv(q, k, v)
    B, H, Sq, D = q.shape
    Skv = k.shape[2]
    for name, t, n in (("q_seg", q_seg, Sq), ("kv_seg", kv_seg, Skv)):
        if (not isinstance(t, torch.Tensor) or t.dtype != torch.int32 or tuple(t.shape) != (B, n)
                or t.device != q.device or not t.is_contiguous()):
            raise TypeError(f"{name} must be a contiguous int32 CUDA tensor of shape [{B}, {n}] on q's device")
    scale = 1.0 / math.sqrt(D) if scale is None else float(scale)
    out, lse = _outputs(q, out, lse, return_lse)
    with torch.cuda.device(q.device):
        st = load().vdx_attn_fwd_segments(q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(),
                                          lse.data_ptr() if lse is not None else None,
                                          B, H, Sq, Skv, D, q_seg.data_ptr(), kv_seg.data_ptr(), scale,
                                          _stream_handle(q.device))
    if st != VDX_OK:
        raise VdxError(st, "vdx_attn_fwd_segments")
    return out, lse


def rope3d(x, grid, s0, dims, theta, interleaved=True, out=None):
    """3D rotary position embedding through ``vdx_rope3d``.

    x: bf16 CUDA tensor [B,H,S,D]; grid = (F, Hp, Wp): tokens [s0, s0 + F*Hp*Wp)
    are the video grid in raster order; dims = (d_t, d_h, d_w).  out=x rotates
    in place; out=None allocates the result.  Returns out.
    """
    if not isinstance(x, torch.Tensor) or not x.is_cuda or x.dtype != torch.bfloat16 or x.dim() != 4 \
            or not x.is_contiguous():
        raise TypeError("x must be a contiguous bf16 CUDA tensor [B,H,S,D]")
    if out is None:
        out = torch.empty_like(x)
    elif out.shape != x.shape or out.dtype != x.dtype or not out.is_contiguous() or out.device != x.device:
        raise ValueError("out must be a contiguous bf16 tensor shaped like x on x's device")
    B, H, S, D = x.shape
    F, Hp, Wp = (int(v) for v in grid)
    d_t, d_h, d_w = (int(v) for v in dims)
    with torch.cuda.device(x.device):
        st = load().vdx_rope3d(x.data_ptr(), out.data_ptr(), B, H, S, D, F, Hp, Wp, int(s0), d_t, d_h, d_w,
                               float(theta), int(bool(interleaved)), _stream_handle(x.device))
    if st != VDX_OK:
        raise VdxError(st, "vdx_rope3d")
    return out


def attn_fwd_rope3d(q, k, v, grid, s0, dims, theta, interleaved=True, scale=None, out=None, lse=None,
                    return_lse=True):
    """Self-attention with the 3D RoPE of q and k, through ``vdx_attn_fwd_rope3d``:
    bit for bit rope3d(q), rope3d(k), then attn_fwd, with the turned tensors in
    library buffers; q and k unchanged.

    q, k, v: bf16 [B,H,S,D] (CUDA); grid = (F, Hp, Wp); dims = (d_t, d_h, d_w).
    """
    _check_qkv(q, k, v)
    B, H, S, D = q.shape
    if k.shape[2] != S:
        raise ValueError("q and k must hold the same tokens")
    F, Hp, Wp = (int(x) for x in grid)
    d_t, d_h, d_w = (int(x) for x in dims)
    scale = 1.0 / math.sqrt(D) if scale is None else float(scale)
    out, lse = _outputs(q, out, lse, return_lse)
    with torch.cuda.device(q.device):
        st = load().vdx_attn_fwd_rope3d(q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(),
                                        lse.data_ptr() if lse is not None else None, B, H, S, D, F, Hp, Wp,
                                        int(s0), d_t, d_h, d_w, float(theta), int(bool(interleaved)), scale,
                                        _stream_handle(q.device))
    if st != VDX_OK:
        raise VdxError(st, "vdx_attn_fwd_rope3d")
    return out, lse


def attn_fwd_win3d(q, k, v, grid, window, neighbourhood=True, scale=None, out=None, lse=None, return_lse=True):
    """Windowed 3D attention through ``vdx_attn_fwd_win3d``.

    q, k, v: bf16 [B,H,S,D] with S = F*Hp*Wp tokens of grid = (F, Hp, Wp) in
    raster order; window = (kt, kh, kw), odd sizes.
    """
    _check_qkv(q, k, v)
    B, H, S, D = q.shape
    F, Hp, Wp = (int(x) for x in grid)
    if S != F * Hp * Wp or k.shape[2] != S:
        raise ValueError(f"q, k, v must hold the F*Hp*Wp = {F * Hp * Wp} grid tokens")
    scale = 1.0 / math.sqrt(D) if scale is None else float(scale)
    out, lse = _outputs(q, out, lse, return_lse)
    with torch.cuda.device(q.device):
        st = load().vdx_attn_fwd_win3d(q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(),
                                       lse.data_ptr() if lse is not None else None, B, H, F, Hp, Wp, D,
                                       int(window[0]), int(window[1]), int(window[2]), int(bool(neighbourhood)),
                                       scale, _stream_handle(q.device))
    if st != VDX_OK:
        raise VdxError(st, "vdx_attn_fwd_win3d")
    return out, lse


def _host_check(q, k, v):
    """Checks CPU q, k, v."""
    for name, t in (("q", q), ("k", k), ("v", v)):
        if not isinstance(t, torch.Tensor) or t.device.type != "cpu":
            raise TypeError(f"{name} must be a CPU tensor")
        if t.dtype != torch.bfloat16 or t.dim() != 4 or not t.is_contiguous():
            raise TypeError(f"{name} must be a contiguous bf16 [B,H,S,D] tensor")
    if k.shape != v.shape or q.shape[:2] != k.shape[:2] or q.shape[3] != k.shape[3]:
        raise ValueError(f"shape mismatch q{tuple(q.shape)} k{tuple(k.shape)} v{tuple(v.shape)}")


def _host_outputs(q, out, lse, return_lse):
    """Makes (or checks) the CPU outputs: pinned when made here."""
    B, H, Sq, D = q.shape
    if out is None:
        out = torch.empty(q.shape, dtype=torch.bfloat16, pin_memory=True)
    elif (out.device.type != "cpu" or out.shape != q.shape or out.dtype != torch.bfloat16
          or not out.is_contiguous()):
        raise ValueError("out must be a contiguous bf16 CPU tensor shaped like q")
    if lse is None and return_lse:
        lse = torch.empty((B, H, Sq), dtype=torch.float32, pin_memory=True)
    elif lse is not None and (lse.device.type != "cpu" or lse.shape != (B, H, Sq)
                              or lse.dtype != torch.float32 or not lse.is_contiguous()):
        raise ValueError("lse must be a contiguous fp32 [B,H,Sq] CPU tensor")
    return out, lse


def _host_ints(x, shape, name):
    if (not isinstance(x, torch.Tensor) or x.device.type != "cpu" or x.dtype != torch.int32
            or tuple(x.shape) != tuple(shape) or not x.is_contiguous()):
        raise TypeError(f"{name} must be a contiguous int32 CPU tensor of shape {list(shape)}")


def _host_call(fn, name, args, device, synchronize):
    device = torch.device("cuda", torch.cuda.current_device()) if device is None else torch.device(device)
    with torch.cuda.device(device):
        st = fn(*args, _stream_handle(device))
        if st != VDX_OK:
            raise VdxError(st, name)
        if synchronize:
            torch.cuda.current_stream(device).synchronize()


def attn_fwd_host(q, k, v, kv_lens=None, scale=None, out=None, lse=None, return_lse=True, chunk_rows=0,
                  device=None, synchronize=True):
    """Attention forward on host tensors through ``vdx_attn_fwd_host``.

    q: bf16 [B,H,Sq,D]; k, v: bf16 [B,H,Skv,D]; kv_lens: optional int32 [B]
    (valid key counts, as attn_fwd_varlen).  All CPU tensors, contiguous;
    pinned memory lets the library overlap the copies with the kernel.
    out / lse default to new pinned CPU tensors.  The call is enqueued on the
    current stream of `device` (default: the current CUDA device); with
    synchronize=False the results are complete only once that stream is
    synchronised.  Returns (out, lse or None).
    """
    _host_check(q, k, v)
    B, H, Sq, D = q.shape
    if kv_lens is not None:
        _host_ints(kv_lens, (B,), "kv_lens")
    out, lse = _host_outputs(q, out, lse, return_lse)
    scale = 1.0 / math.sqrt(D) if scale is None else float(scale)
    _host_call(load().vdx_attn_fwd_host, "vdx_attn_fwd_host",
               (q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(),
                lse.data_ptr() if lse is not None else None, B, H, Sq, k.shape[2], D,
                kv_lens.data_ptr() if kv_lens is not None else None, scale, int(chunk_rows)), device, synchronize)
    return out, lse


def attn_fwd_segments_host(q, k, v, q_seg, kv_seg, scale=None, out=None, lse=None, return_lse=True, chunk_rows=0,
                           device=None, synchronize=True):
    """Joint attention with segment ids on host tensors through
    ``vdx_attn_fwd_segments_host``; q_seg int32 [B, Sq], kv_seg int32 [B, Skv]
    (CPU).  Other arguments as attn_fwd_host."""
    _host_check(q, k, v)
    B, H, Sq, D = q.shape
    Skv = k.shape[2]
    _host_ints(q_seg, (B, Sq), "q_seg")
    _host_ints(kv_seg, (B, Skv), "kv_seg")
    out, lse = _host_outputs(q, out, lse, return_lse)
    scale = 1.0 / math.sqrt(D) if scale is None else float(scale)
    _host_call(load().vdx_attn_fwd_segments_host, "vdx_attn_fwd_segments_host",
               (q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(),
                lse.data_ptr() if lse is not None else None, B, H, Sq, Skv, D, q_seg.data_ptr(),
                kv_seg.data_ptr(), scale, int(chunk_rows)), device, synchronize)
    return out, lse


def attn_fwd_win3d_host(q, k, v, grid, window, neighbourhood=True, scale=None, out=None, lse=None,
                        return_lse=True, chunk_rows=0, device=None, synchronize=True):
    """Windowed 3D attention on host tensors through ``vdx_attn_fwd_win3d_host``;
    grid = (F, Hp, Wp), window = (kt, kh, kw) as attn_fwd_win3d.  Other
    arguments as attn_fwd_host."""
    _host_check(q, k, v)
    B, H, S, D = q.shape
    F, Hp, Wp = (int(x) for x in grid)
    if S != F * Hp * Wp or k.shape[2] != S:
        raise ValueError(f"q, k, v must hold the F*Hp*Wp = {F * Hp * Wp} grid tokens")
    out, lse = _host_outputs(q, out, lse, return_lse)
    scale = 1.0 / math.sqrt(D) if scale is None else float(scale)
    _host_call(load().vdx_attn_fwd_win3d_host, "vdx_attn_fwd_win3d_host",
               (q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(),
                lse.data_ptr() if lse is not None else None, B, H, F, Hp, Wp, D, int(window[0]), int(window[1]),
                int(window[2]), int(bool(neighbourhood)), scale, int(chunk_rows)), device, synchronize)
    return out, lse


def attn_fwd_rope3d_host(q, k, v, grid, s0, dims, theta, interleaved=True, scale=None, out=None, lse=None,
                         return_lse=True, chunk_rows=0, device=None, synchronize=True):
    """attn_fwd_rope3d on host tensors through ``vdx_attn_fwd_rope3d_host``
    (each chunk's q and k rows turned in the device slot, then attended).
    Other arguments as attn_fwd_host."""
    _host_check(q, k, v)
    B, H, S, D = q.shape
    if k.shape[2] != S:
        raise ValueError("q and k must hold the same tokens")
    F, Hp, Wp = (int(x) for x in grid)
    d_t, d_h, d_w = (int(x) for x in dims)
    out, lse = _host_outputs(q, out, lse, return_lse)
    scale = 1.0 / math.sqrt(D) if scale is None else float(scale)
    _host_call(load().vdx_attn_fwd_rope3d_host, "vdx_attn_fwd_rope3d_host",
               (q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(),
                lse.data_ptr() if lse is not None else None, B, H, S, D, F, Hp, Wp, int(s0), d_t, d_h, d_w,
                float(theta), int(bool(interleaved)), scale, int(chunk_rows)), device, synchronize)
    return out, lse
