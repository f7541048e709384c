"""GB300-native (sm_103a) softmax attention forward for video-DiT inference.

The compute path is the CUDA library ``_lib/libvdx.so`` (C ABI in
``include/vdx.h``); ``binding`` forwards torch tensors' device pointers to
it.  The library is loaded on first use and its absence is an error.
"""
from .binding import (VdxError, attn_fwd, attn_fwd_host, attn_fwd_rope3d, attn_fwd_rope3d_host,  # noqa: F401
                      attn_fwd_segments, attn_fwd_segments_host, attn_fwd_varlen, attn_fwd_win3d,
                      attn_fwd_win3d_host, check_device_error, load, release, rope3d, selftest_wait_timeout,
                      status_string, version)
