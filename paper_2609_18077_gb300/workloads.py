"""Seeded synthetic attention workloads shaped like the paper's video DiTs.

This module only draws inputs; it holds none of the attention arithmetic and
is the one piece shared by the CUDA path's tests and the CPU oracle.

Geometry: a latent video of F x Hp x Wp patches flattened to S = F*Hp*Wp
tokens per sample (vidax paper, Sec. 1: patchifying temporal volumes gives
sequences of tens of thousands of tokens; the Wan2.1 832x480 and 1280x720,
81-frame rows of Table 5 give 21x30x52 and 21x45x80 latents).  Cross-attention
attends video tokens to a padded batch of text tokens with per-sample valid
lengths (Sec. 3.1, Wan's UMT5 text conditioning; appendix Table 4 on masking
padded text tokens).  Classifier-free guidance doubles the internal batch
(Sec. 4, experimental setup), hence B = 2 for the text cross-attention.

Recipe (every draw is seeded; no dataset is read):
  * rng = numpy PCG64(seed); Q, K, V ~ N(0, 1) float32, drawn in that order;
  * "logit std ~ 3": Q and K are multiplied by sqrt(3) in float32 before the
    bf16 cast, so with scale = 1/sqrt(D) the logits scale*q.k have std ~ 3;
  * cast to bf16 by round-to-nearest-even (torch CPU);
  * outlier keys: per sample, round(frac * Skv) token positions drawn without
    replacement (shared by all heads), those K rows multiplied by 8 after the
    cast (exact: a power of two);
  * text lengths: one integer per sample, uniform on the inclusive range
    [lo, hi]; K/V rows past a sample's length are padding and may be filled
    with NaN to prove they are never read;
  * row subsets for large configs: per (b, h), n distinct query rows;
  * windowed 3D attention (appendix Table 4: the LTX-2.5 VAE decoder's
    neighbourhood attention with an 11^3 window): the win3d workload's tokens
    are a 16x32x48 grid in raster order (t, h, w), each query attending the
    11x11x11 window around it (shifted inward at the border); the decoder's
    shapes are not in the paper, so H = 8 and D = 128 are our choice;
  * 3D RoPE (Sec. 2: each family keeps its own convention): the rope480
    workload rotates small480's Q and K over its 21x30x52 grid with Wan's
    published split (44/42/42 head dims for t/h/w, interleaved pairs,
    theta = 1e4) before the attention;
  * joint text-video attention (appendix Table 4, HunyuanVideo-1.5's joint
    attention over video and padded text, masked through segment ids; the
    ~45k-token CogVideoX1.5 joint sequence of Table 3): each sample is
    text_slots text tokens followed by the video tokens; a sample's valid text
    length is uniform on the inclusive range [lo, hi]; segment id 1 marks the
    valid text and every video token, 0 the padded text slots, for queries
    and keys alike (self-attention over one sequence).
Independent streams (lengths, outliers, row subsets, joint text lengths) come from
SeedSequence(seed).spawn so that adding one never shifts another.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np
import torch

BF16_NAN_BITS = 0x7FC0


@dataclass(frozen=True)
class Workload:
    """One attention problem: shapes plus the recipe of its synthetic inputs."""
    name: str
    B: int
    H: int
    D: int
    Sq: int
    Skv: int
    seed: int
    latent: tuple = ()            # (frames, rows, cols) of patches, when Sq comes from one
    logit_gain: float = 1.0       # Q and K are scaled by this before the bf16 cast
    outlier_frac: float = 0.0     # fraction of K rows multiplied by 8
    kv_len_range: tuple | None = None   # inclusive (lo, hi) per-sample text lengths
    oracle_rows: int | None = None      # per (b, h) query rows the parity check compares
    joint_text: tuple | None = None     # (text_slots, lo, hi): joint text-video segments
    rope: tuple | None = None           # ((F, Hp, Wp), s0, (d_t, d_h, d_w), theta, interleaved) on Q and K
    window: tuple | None = None         # ((kt, kh, kw), neighbourhood): windowed attention over the latent grid
    description: str = field(default="", compare=False)

    @property
    def scale(self) -> float:
        return 1.0 / math.sqrt(self.D)

    @property
    def varlen(self) -> bool:
        return self.kv_len_range is not None

    @property
    def segments(self) -> bool:
        return self.joint_text is not None

    def flops(self, kv_lens=None, q_seg=None, kv_seg=None) -> float:
        """Algorithmic FLOPs 4*B*H*Sq*Skv*D (two GEMMs, 2 flops per MAC).

        With kv_lens the effective count uses the valid keys of each sample;
        with segment ids, the (query, key) pairs that share a segment.
        """
        if q_seg is not None:
            return 4.0 * self.H * self.D * float(segment_pairs(q_seg, kv_seg))
        if self.window is not None:
            return 4.0 * self.B * self.H * self.D * float(window_pairs(self.latent, *self.window))
        if kv_lens is None:
            return 4.0 * self.B * self.H * self.Sq * self.Skv * self.D
        return 4.0 * self.H * self.Sq * self.D * float(np.sum(np.clip(kv_lens, 0, self.Skv)))


WORKLOADS = {
    "tiny": Workload(
        "tiny", B=1, H=2, D=64, Sq=192, Skv=192, seed=1001, latent=(3, 8, 8),
        description="tiny self-attention, latent 3x8x8 -> 192 tokens"),
    "small480": Workload(
        "small480", B=1, H=12, D=128, Sq=32760, Skv=32760, seed=1002, latent=(21, 30, 52),
        logit_gain=math.sqrt(3.0), oracle_rows=4096,
        description="small-DiT 480p self-attention, latent 21x30x52 -> 32760 tokens, logit std ~3"),
    "cross": Workload(
        "cross", B=2, H=12, D=128, Sq=32760, Skv=512, seed=1003, latent=(21, 30, 52),
        kv_len_range=(64, 512),
        description="video-to-text cross-attention, 32760 video tokens x <=512 text tokens, CFG batch 2"),
    "large480": Workload(
        "large480", B=1, H=40, D=128, Sq=32760, Skv=32760, seed=1004, latent=(21, 30, 52),
        logit_gain=math.sqrt(3.0), outlier_frac=0.05, oracle_rows=4096,
        description="large-DiT 480p self-attention, logit std ~3, 5% outlier key rows x8"),
    "large720": Workload(
        "large720", B=1, H=40, D=128, Sq=75600, Skv=75600, seed=1005, latent=(21, 45, 80),
        oracle_rows=4096,
        description="large-DiT 720p self-attention, latent 21x45x80 -> 75600 tokens"),
    "large720_h4": Workload(
        "large720_h4", B=1, H=4, D=128, Sq=75600, Skv=75600, seed=1005, latent=(21, 45, 80),
        oracle_rows=4096,
        description="large720's sequence with 4 heads: the same kernel and unit length at a tenth of the "
                    "device memory, for multi-pass profiler captures"),
    "rope480": Workload(
        "rope480", B=1, H=12, D=128, Sq=32760, Skv=32760, seed=1002, latent=(21, 30, 52),
        logit_gain=math.sqrt(3.0), oracle_rows=4096,
        rope=((21, 30, 52), 0, (44, 42, 42), 10000.0, True),
        description="small480 with a 3D rotary embedding of Q and K (Wan-style: 44/42/42 dims of t/h/w, "
                    "interleaved pairs, theta 1e4) before the attention"),
    "win3d": Workload(
        "win3d", B=1, H=8, D=128, Sq=24576, Skv=24576, seed=1007, latent=(16, 32, 48),
        window=((11, 11, 11), True), oracle_rows=4096,
        description="3D neighbourhood attention with an 11x11x11 window over a 16x32x48 latent grid "
                    "(the LTX-2.5 VAE decoder's windowed attention; shapes are not in the paper)"),
    "joint45k": Workload(
        "joint45k", B=2, H=48, D=64, Sq=45106, Skv=45106, seed=1006, latent=(11, 48, 85),
        joint_text=(226, 16, 226), oracle_rows=4096,
        description="joint text-video self-attention, 226 text slots + latent 11x48x85 = 44880 video "
                    "tokens, padded text masked by segment ids, CFG batch 2, D=64"),
}

# The bench's default workload: the largest single-GPU configuration, the
# large-DiT 720p self-attention (B=1, H=40, D=128, S = 21*45*80 = 75600).
DEFAULT_WORKLOAD = "large720"


def _spawn(seed: int, n: int = 4):
    return [np.random.Generator(np.random.PCG64(s)) for s in np.random.SeedSequence(seed).spawn(n)]


def to_bf16(a: np.ndarray) -> torch.Tensor:
    """float32 numpy -> bf16 torch CPU tensor (round to nearest even)."""
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(torch.bfloat16)


def bf16_bits(t: torch.Tensor) -> np.ndarray:
    """bf16 torch tensor -> numpy uint16 bit patterns (same shape, CPU copy)."""
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def random_qkv(B, H, Sq, Skv, D, seed, logit_gain=1.0):
    """Q, K, V as bf16 CPU tensors, N(0,1) with Q and K scaled by logit_gain."""
    rng = np.random.Generator(np.random.PCG64(seed))
    q = rng.standard_normal((B, H, Sq, D), dtype=np.float32)
    k = rng.standard_normal((B, H, Skv, D), dtype=np.float32)
    v = rng.standard_normal((B, H, Skv, D), dtype=np.float32)
    if logit_gain != 1.0:
        g = np.float32(logit_gain)
        q *= g
        k *= g
    return to_bf16(q), to_bf16(k), to_bf16(v)


def draw_kv_lens(B, lo, hi, seed) -> np.ndarray:
    """Per-sample valid key counts, uniform on the inclusive range [lo, hi]."""
    rng = _spawn(seed)[0]
    return rng.integers(lo, hi + 1, size=B, dtype=np.int64).astype(np.int32)


def draw_outlier_rows(B, Skv, frac, seed) -> list:
    """Per sample, round(frac*Skv) distinct key positions (sorted)."""
    rng = _spawn(seed)[1]
    n = int(round(frac * Skv))
    return [np.sort(rng.choice(Skv, size=n, replace=False)) for _ in range(B)]


def draw_rows(B, H, Sq, n, seed) -> np.ndarray:
    """Per (b, h), n distinct query rows (sorted), shape [B*H, n] int32."""
    rng = _spawn(seed)[2]
    n = min(n, Sq)
    return np.stack([np.sort(rng.choice(Sq, size=n, replace=False)) for _ in range(B * H)]).astype(np.int32)


def draw_text_lens(B, lo, hi, seed) -> np.ndarray:
    """Per-sample valid text lengths of a joint sequence, uniform on [lo, hi]."""
    rng = _spawn(seed)[3]
    return rng.integers(lo, hi + 1, size=B, dtype=np.int64).astype(np.int32)


def joint_segments(text_lens, text_slots, S) -> np.ndarray:
    """Segment ids [B, S] int32 of joint sequences: text_slots text tokens, then
    video tokens; 1 for valid text and video, 0 for padded text slots."""
    seg = np.ones((len(text_lens), S), dtype=np.int32)
    for b, L in enumerate(np.asarray(text_lens)):
        seg[b, int(L):text_slots] = 0
    return seg


def window_pairs(grid, window, neighbourhood) -> int:
    """Number of (query, key) pairs inside the windows of one sequence."""
    total = 1
    for L, k in zip(grid, window):
        p = np.arange(L)
        if neighbourhood:
            n = min(k, L)
            total *= n * L
            continue
        lo = np.maximum(p - k // 2, 0)
        hi = np.minimum(p + k // 2, L - 1)
        total *= int(np.sum(hi - lo + 1))
    return int(total)


def segment_pairs(q_seg, kv_seg) -> int:
    """Number of (query, key) pairs with equal segment ids, summed over samples."""
    total = 0
    for qs, ks in zip(np.asarray(q_seg), np.asarray(kv_seg)):
        ids, qn = np.unique(qs, return_counts=True)
        kid, kn = np.unique(ks, return_counts=True)
        common, qi, ki = np.intersect1d(ids, kid, return_indices=True)
        total += int(np.sum(qn[qi].astype(np.int64) * kn[ki].astype(np.int64)))
    return total


def pad_invalid_keys(k: torch.Tensor, v: torch.Tensor, kv_lens, fill_bits: int = BF16_NAN_BITS):
    """Overwrite K/V rows past each sample's valid length with a bf16 bit pattern."""
    k = k.clone()
    v = v.clone()
    kb = k.view(torch.int16)
    vb = v.view(torch.int16)
    fill = np.array(fill_bits, dtype=np.uint16).view(np.int16).item()
    for b, L in enumerate(np.asarray(kv_lens)):
        L = int(max(0, min(int(L), k.shape[2])))
        kb[b, :, L:, :] = fill
        vb[b, :, L:, :] = fill
    return k, v


def generate(w: Workload | str, nan_padding: bool = True):
    """Materialise a workload on the CPU.

    Returns a dict with q, k, v (bf16 CPU tensors [B,H,S,D]), scale,
    kv_lens (int32 numpy [B] or None), rows (int32 [B*H, n] or None: the
    query rows a parity check compares), q_seg / kv_seg (int32 numpy
    [B,Sq] / [B,Skv] segment ids, or None) and the workload itself.
    """
    if isinstance(w, str):
        w = WORKLOADS[w]
    q, k, v = random_qkv(w.B, w.H, w.Sq, w.Skv, w.D, w.seed, w.logit_gain)
    if w.outlier_frac > 0:
        for b, idx in enumerate(draw_outlier_rows(w.B, w.Skv, w.outlier_frac, w.seed)):
            k[b, :, torch.from_numpy(idx.astype(np.int64)), :] *= 8
    kv_lens = None
    if w.kv_len_range is not None:
        kv_lens = draw_kv_lens(w.B, w.kv_len_range[0], w.kv_len_range[1], w.seed)
        if nan_padding:
            k, v = pad_invalid_keys(k, v, kv_lens)
    q_seg = kv_seg = None
    if w.joint_text is not None:
        slots, lo, hi = w.joint_text
        seg = joint_segments(draw_text_lens(w.B, lo, hi, w.seed), slots, w.Sq)
        q_seg = kv_seg = seg
    rows = None
    if w.oracle_rows is not None and w.oracle_rows < w.Sq:
        rows = draw_rows(w.B, w.H, w.Sq, w.oracle_rows, w.seed)
    return {"workload": w, "q": q, "k": k, "v": v, "scale": w.scale,
            "kv_lens": kv_lens, "rows": rows, "q_seg": q_seg, "kv_seg": kv_seg}
