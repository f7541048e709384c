"""Pins of the fp64 oracle to facts other than itself.

Each pin takes an ``oracle.Oracle`` handle and raises AssertionError when the
oracle disagrees with a closed form, an invariant of softmax attention, an
independent library routine or a high-precision brute-force evaluation.
``test_oracle.py`` runs them on the real oracle; ``test_oracle_mutants.py``
runs them on copies of the oracle with planted mistakes and requires every
mistake to be caught by at least one pin.

Sources of the facts (none of them is the oracle's own code):
  * closed forms of softmax attention with one or two keys;
  * invariants: weights sum to one, constant values are returned unchanged,
    query-row permutation equivariance, joint key/value permutation
    invariance, translation of values, zero logits give the mean;
  * masking: a sample with L valid keys equals dense attention on the first
    L keys, whatever the padding holds (appendix Table 4 of the paper:
    padded text tokens must not be attended);
  * segment ids (joint text-video attention, same appendix entry): one
    segment everywhere is dense attention; packed segments are independent
    problems; a prefix segment is the valid-count form; torch's SDPA with the
    boolean mask q_seg[i] == kv_seg[j];
  * windowed 3D attention: torch SDPA with the window mask (each border rule
    characterised independently), whole-grid windows as dense attention, a
    1x1x1 window, window sizes, interior agreement of the two rules;
  * 3D RoPE: the textbook complex form z exp(i phi), norm preservation,
    identity off the grid and at its origin, one axis per coordinate, dot
    products depending on relative position only, and the two pairings
    agreeing up to a permutation of dims;
  * torch's scaled_dot_product_attention and logsumexp in fp64 (a library);
  * a 50-digit mpmath evaluation on a tiny input.
"""
from __future__ import annotations

import math

import numpy as np
import torch

from paper_2609_18077_gb300.workloads import bf16_bits, random_qkv, to_bf16, pad_invalid_keys

TOL = 1e-12


def _dec(bits) -> np.ndarray:
    """bf16 bit patterns -> float64 (exact), independent of the oracle."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def _bits_of(values) -> np.ndarray:
    return bf16_bits(to_bf16(np.asarray(values, dtype=np.float32)))


def _inputs(B, H, Sq, Skv, D, seed, gain=1.0):
    q, k, v = random_qkv(B, H, Sq, Skv, D, seed, gain)
    return bf16_bits(q), bf16_bits(k), bf16_bits(v)


def pin_single_key(orc):
    """Skv = 1: o = v_0 exactly and lse = scale * q.k_0."""
    q, k, v = _inputs(2, 3, 5, 1, 16, seed=11)
    scale = 0.37
    o, lse = orc.attn_fwd(q, k, v, scale)
    qd, kd, vd = _dec(q), _dec(k), _dec(v)
    np.testing.assert_allclose(o, np.broadcast_to(vd, o.shape), rtol=0, atol=TOL)
    want = scale * np.einsum("bhid,bhjd->bhi", qd, kd)
    np.testing.assert_allclose(lse, want, rtol=TOL, atol=TOL)


def pin_two_keys(orc):
    """Skv = 2: o = (1-w) v_0 + w v_1 with w = sigmoid(s_1 - s_0); lse = log(e^s0 + e^s1)."""
    q, k, v = _inputs(1, 2, 7, 2, 8, seed=12)
    scale = 0.8
    o, lse = orc.attn_fwd(q, k, v, scale)
    qd, kd, vd = _dec(q), _dec(k), _dec(v)
    s = scale * np.einsum("bhid,bhjd->bhij", qd, kd)
    w = 1.0 / (1.0 + np.exp(s[..., 0] - s[..., 1]))
    want_o = (1 - w)[..., None] * vd[:, :, 0:1, :] + w[..., None] * vd[:, :, 1:2, :]
    np.testing.assert_allclose(o, want_o, rtol=0, atol=1e-12)
    hi = np.maximum(s[..., 0], s[..., 1])
    want_lse = hi + np.log1p(np.exp(-np.abs(s[..., 0] - s[..., 1])))
    np.testing.assert_allclose(lse, want_lse, rtol=TOL, atol=TOL)


def pin_weights_sum_to_one(orc):
    """Softmax weights are non-negative and every row sums to one; o = P @ V."""
    q, k, v = _inputs(2, 2, 9, 13, 16, seed=13, gain=2.0)
    o, lse, p = orc.attn_fwd(q, k, v, 0.25, probs=True)
    assert np.all(p >= 0)
    np.testing.assert_allclose(p.sum(-1), 1.0, rtol=0, atol=1e-13)
    np.testing.assert_allclose(o, p @ _dec(v), rtol=0, atol=1e-12)


def pin_constant_values(orc):
    """If every value row is the same vector c, the output is c."""
    q, k, _ = _inputs(1, 2, 6, 11, 8, seed=14, gain=3.0)
    c = np.array([1.5, -2.0, 0.25, 3.0, -0.125, 7.0, 0.0, -1.0], dtype=np.float32)
    v = _bits_of(np.broadcast_to(c, (1, 2, 11, 8)))
    o, _ = orc.attn_fwd(q, k, v, 0.5)
    np.testing.assert_allclose(o, np.broadcast_to(c.astype(np.float64), o.shape), rtol=0, atol=1e-12)


def pin_zero_logits(orc):
    """scale = 0 (or q = 0): every weight is 1/L, o = mean of the L values, lse = ln L."""
    q, k, v = _inputs(2, 2, 4, 10, 8, seed=15)
    for case in ("scale", "q"):
        if case == "scale":
            o, lse = orc.attn_fwd(q, k, v, 0.0)
        else:
            o, lse = orc.attn_fwd(np.zeros_like(q), k, v, 0.9)
        want = _dec(v).mean(axis=2, keepdims=True)
        np.testing.assert_allclose(o, np.broadcast_to(want, o.shape), rtol=0, atol=1e-13)
        np.testing.assert_allclose(lse, math.log(10), rtol=0, atol=1e-13)


def pin_query_permutation(orc):
    """Permuting query rows permutes o and lse the same way."""
    q, k, v = _inputs(1, 2, 12, 9, 16, seed=16, gain=1.5)
    perm = np.random.default_rng(1).permutation(12)
    o, lse = orc.attn_fwd(q, k, v, 0.3)
    o2, lse2 = orc.attn_fwd(np.ascontiguousarray(q[:, :, perm]), k, v, 0.3)
    np.testing.assert_array_equal(o2, o[:, :, perm])
    np.testing.assert_array_equal(lse2, lse[:, :, perm])


def pin_key_value_permutation(orc):
    """Permuting key rows and value rows jointly changes nothing (up to rounding)."""
    q, k, v = _inputs(2, 1, 5, 17, 8, seed=17, gain=1.5)
    perm = np.random.default_rng(2).permutation(17)
    o, lse = orc.attn_fwd(q, k, v, 0.4)
    o2, lse2 = orc.attn_fwd(q, np.ascontiguousarray(k[:, :, perm]), np.ascontiguousarray(v[:, :, perm]), 0.4)
    np.testing.assert_allclose(o2, o, rtol=0, atol=1e-13)
    np.testing.assert_allclose(lse2, lse, rtol=1e-14, atol=1e-13)


def pin_value_translation(orc):
    """Adding a constant row c to every value adds c to the output (weights sum to one)."""
    # small integers keep v + c exactly representable in bf16
    rng = np.random.default_rng(3)
    q, k, _ = _inputs(1, 2, 5, 7, 4, seed=18)
    vi = rng.integers(-8, 9, size=(1, 2, 7, 4)).astype(np.float32)
    c = np.array([3.0, -5.0, 1.0, 16.0], dtype=np.float32)
    o1, _ = orc.attn_fwd(q, k, _bits_of(vi), 0.6)
    o2, _ = orc.attn_fwd(q, k, _bits_of(vi + c), 0.6)
    np.testing.assert_allclose(o2 - o1, np.broadcast_to(c.astype(np.float64), o1.shape), rtol=0, atol=1e-12)


def pin_varlen_is_truncation(orc):
    """L valid keys (NaN padding after them) equal dense attention over the first L keys."""
    B, H, Sq, Skv, D = 3, 2, 6, 20, 8
    q, k, v = random_qkv(B, H, Sq, Skv, D, seed=19, logit_gain=1.2)
    lens = np.array([20, 7, 1], dtype=np.int32)
    kp, vp = pad_invalid_keys(k, v, lens)
    o, lse = orc.attn_fwd(bf16_bits(q), bf16_bits(kp), bf16_bits(vp), 0.35, kv_lens=lens)
    assert np.all(np.isfinite(o))
    for b, L in enumerate(lens):
        ob, lb = orc.attn_fwd(bf16_bits(q[b:b + 1]), bf16_bits(k[b:b + 1, :, :L]),
                              bf16_bits(v[b:b + 1, :, :L]), 0.35)
        np.testing.assert_array_equal(o[b:b + 1], ob)
        np.testing.assert_array_equal(lse[b:b + 1], lb)


def pin_varlen_empty_and_clamped(orc):
    """L = 0 gives o = 0, lse = -inf; lengths beyond Skv clamp to Skv; negative to 0."""
    q, k, v = _inputs(3, 1, 4, 5, 8, seed=20)
    o, lse = orc.attn_fwd(q, k, v, 0.5, kv_lens=[0, 99, -3])
    assert np.all(o[0] == 0) and np.all(np.isneginf(lse[0]))
    assert np.all(o[2] == 0) and np.all(np.isneginf(lse[2]))
    od, ld = orc.attn_fwd(q[1:2], k[1:2], v[1:2], 0.5)
    np.testing.assert_array_equal(o[1:2], od)
    np.testing.assert_array_equal(lse[1:2], ld)


def pin_row_subset(orc):
    """A row subset returns exactly the full result at those rows, per (b, h)."""
    q, k, v = _inputs(2, 2, 11, 9, 8, seed=21)
    rows = np.array([[10, 0, 3], [1, 2, 9], [5, 5, 7], [0, 10, 4]], dtype=np.int32)
    o, lse = orc.attn_fwd(q, k, v, 0.7)
    os_, ls = orc.attn_fwd(q, k, v, 0.7, rows=rows)
    of = o.reshape(4, 11, 8)
    lf = lse.reshape(4, 11)
    for bh in range(4):
        np.testing.assert_array_equal(os_.reshape(4, 3, 8)[bh], of[bh, rows[bh]])
        np.testing.assert_array_equal(ls.reshape(4, 3)[bh], lf[bh, rows[bh]])


def pin_torch_sdpa(orc):
    """torch scaled_dot_product_attention and logsumexp in fp64 on the CPU (a library)."""
    for (B, H, Sq, Skv, D, scale, seed) in [(1, 2, 17, 33, 64, 0.125, 22),
                                             (2, 3, 40, 9, 128, 0.2, 23),
                                             (1, 1, 5, 64, 16, -0.3, 24)]:
        q, k, v = random_qkv(B, H, Sq, Skv, D, seed, logit_gain=1.7)
        o, lse = orc.attn_fwd(bf16_bits(q), bf16_bits(k), bf16_bits(v), scale)
        qd, kd, vd = q.double(), k.double(), v.double()
        want = torch.nn.functional.scaled_dot_product_attention(qd, kd, vd, scale=scale)
        want_lse = torch.logsumexp(scale * (qd @ kd.transpose(-1, -2)), dim=-1)
        np.testing.assert_allclose(o, want.numpy(), rtol=0, atol=1e-12)
        np.testing.assert_allclose(lse, want_lse.numpy(), rtol=1e-13, atol=1e-12)


def pin_mpmath_brute_force(orc):
    """A 50-digit evaluation of the definition on a 1x1x3x4 problem with 4 keys."""
    import mpmath
    mpmath.mp.dps = 50
    q, k, v = _inputs(1, 1, 3, 4, 4, seed=25, gain=2.5)
    scale = 0.45
    o, lse = orc.attn_fwd(q, k, v, scale)
    qd, kd, vd = _dec(q)[0, 0], _dec(k)[0, 0], _dec(v)[0, 0]
    for i in range(3):
        s = [mpmath.mpf(scale) * mpmath.fsum(mpmath.mpf(qd[i, d]) * mpmath.mpf(kd[j, d]) for d in range(4))
             for j in range(4)]
        e = [mpmath.e ** sj for sj in s]
        z = mpmath.fsum(e)
        for d in range(4):
            want = mpmath.fsum(e[j] * mpmath.mpf(vd[j, d]) for j in range(4)) / z
            assert abs(float(want) - o[0, 0, i, d]) <= 1e-14, (i, d)
        assert abs(float(mpmath.log(z)) - lse[0, 0, i]) <= 1e-14


def pin_large_logits_stable(orc):
    """Logits of magnitude ~1000 neither overflow nor underflow (softmax shift invariance)."""
    # q = 32 e_0 and k_j = c_j e_0: exact bf16 inputs with logits spread over 800
    D = 8
    q = np.zeros((1, 1, 1, D), dtype=np.float32)
    q[..., 0] = 32.0
    v = np.zeros((1, 1, 3, D), dtype=np.float32)
    v[0, 0, :, 1] = [1.0, 2.0, 4.0]
    for c in ([-18.75, 0.0, 6.25], [-30.0, -31.0, -31.5]):
        k = np.zeros((1, 1, 3, D), dtype=np.float32)
        k[0, 0, :, 0] = c
        o, lse = orc.attn_fwd(_bits_of(q), _bits_of(k), _bits_of(v), 1.0)
        s = 32.0 * np.array(c)
        w = np.exp(s - s.max())
        want_lse = s.max() + np.log(w.sum())
        w /= w.sum()
        assert np.all(np.isfinite(o)) and np.isfinite(lse).all()
        np.testing.assert_allclose(o[0, 0, 0, 1], (w * [1, 2, 4]).sum(), rtol=0, atol=1e-13)
        np.testing.assert_allclose(lse[0, 0, 0], want_lse, rtol=1e-15, atol=0)


def pin_segments_one_segment_is_dense(orc):
    """Every query and key in one segment (any id): exactly dense attention."""
    q, k, v = _inputs(2, 2, 9, 14, 16, seed=26, gain=1.5)
    o, lse = orc.attn_fwd(q, k, v, 0.3)
    for sid in (0, 7, -4):
        os_, ls = orc.attn_fwd(q, k, v, 0.3, q_seg=np.full((2, 9), sid), kv_seg=np.full((2, 14), sid))
        np.testing.assert_array_equal(os_, o)
        np.testing.assert_array_equal(ls, lse)


def pin_segments_packed_are_independent(orc):
    """Sequences packed into one with distinct segment ids equal separate attention
    over each sequence; a query segment with no key gets o = 0, lse = -inf."""
    B, H, S, D = 2, 2, 15, 8
    q, k, v = _inputs(B, H, S, S, D, seed=27, gain=1.3)
    seg = np.array([[3] * 4 + [5] * 6 + [9] * 5,
                    [1] * 11 + [2] * 4], dtype=np.int32)
    q_seg = seg.copy()
    q_seg[1, 13] = 8          # this query's segment owns no key
    o, lse = orc.attn_fwd(q, k, v, 0.45, q_seg=q_seg, kv_seg=seg)
    for b in range(B):
        for sid in np.unique(seg[b]):
            js = np.flatnonzero(seg[b] == sid)
            lo, hi = js[0], js[-1] + 1
            ob, lb = orc.attn_fwd(q[b:b + 1, :, lo:hi], k[b:b + 1, :, lo:hi], v[b:b + 1, :, lo:hi], 0.45)
            rows = [i for i in range(lo, hi) if q_seg[b, i] == sid]
            np.testing.assert_allclose(o[b][:, rows], ob[0][:, np.array(rows) - lo], rtol=0, atol=1e-14)
            np.testing.assert_allclose(lse[b][:, rows], lb[0][:, np.array(rows) - lo], rtol=1e-15, atol=1e-14)
    assert np.all(o[1, :, 13] == 0) and np.all(np.isneginf(lse[1, :, 13]))


def pin_segments_prefix_is_valid_count(orc):
    """kv_seg = 1 on the first L keys and 0 after (NaN padding), q_seg = 1:
    exactly the valid-count form with kv_lens = L."""
    B, H, Sq, Skv, D = 3, 2, 5, 19, 16
    q, k, v = random_qkv(B, H, Sq, Skv, D, seed=28, logit_gain=1.4)
    lens = np.array([19, 6, 1], dtype=np.int32)
    kp, vp = pad_invalid_keys(k, v, lens)
    kv_seg = (np.arange(Skv)[None, :] < lens[:, None]).astype(np.int32)
    q_seg = np.ones((B, Sq), dtype=np.int32)
    o, lse = orc.attn_fwd(bf16_bits(q), bf16_bits(kp), bf16_bits(vp), 0.25, q_seg=q_seg, kv_seg=kv_seg)
    ov, lv = orc.attn_fwd(bf16_bits(q), bf16_bits(kp), bf16_bits(vp), 0.25, kv_lens=lens)
    assert np.all(np.isfinite(o))
    np.testing.assert_array_equal(o, ov)
    np.testing.assert_array_equal(lse, lv)


def pin_segments_torch_masked_sdpa(orc):
    """Interleaved segment ids against torch SDPA with the boolean mask
    q_seg[i] == kv_seg[j] and a masked logsumexp, fp64 (a library)."""
    B, H, Sq, Skv, D, scale = 2, 3, 21, 26, 32, 0.2
    q, k, v = random_qkv(B, H, Sq, Skv, D, seed=29, logit_gain=1.6)
    rng = np.random.default_rng(30)
    q_seg = rng.integers(0, 3, size=(B, Sq)).astype(np.int32)
    kv_seg = rng.integers(0, 3, size=(B, Skv)).astype(np.int32)
    kv_seg[1, :] = np.where(kv_seg[1, :] == 2, 1, kv_seg[1, :])   # sample 1: segment 2 owns no key
    o, lse, p = orc.attn_fwd(bf16_bits(q), bf16_bits(k), bf16_bits(v), scale, probs=True,
                             q_seg=q_seg, kv_seg=kv_seg)
    mask = torch.from_numpy(q_seg[:, :, None] == kv_seg[:, None, :])[:, None]    # [B,1,Sq,Skv]
    qd, kd, vd = q.double(), k.double(), v.double()
    want = torch.nn.functional.scaled_dot_product_attention(qd, kd, vd, attn_mask=mask, scale=scale)
    logits = (scale * (qd @ kd.transpose(-1, -2))).masked_fill(~mask, -math.inf)
    want_lse = torch.logsumexp(logits, dim=-1)
    has = mask.numpy().any(-1)                                                   # [B,1,Sq]
    has = np.broadcast_to(has, (B, H, Sq))
    assert (~has).any() and has.any()
    np.testing.assert_allclose(o[has], want.numpy()[has], rtol=0, atol=1e-12)
    np.testing.assert_allclose(lse[has], want_lse.numpy()[has], rtol=1e-13, atol=1e-12)
    assert np.all(o[~has] == 0) and np.all(np.isneginf(lse[~has]))
    np.testing.assert_array_equal(p == 0, ~np.broadcast_to(mask.numpy(), p.shape) | (p == 0))
    np.testing.assert_allclose(p.sum(-1)[has], 1.0, rtol=0, atol=1e-13)


# ---- 3D rotary position embedding (Sec. 2: each family keeps its own 3D RoPE convention)

def _rope_x(B, H, S, D, seed, gain=1.0):
    q, _, _ = random_qkv(B, H, S, 1, D, seed, gain)
    return bf16_bits(q)


def pin_rope_complex_rotation(orc):
    """Each pair, read as a complex number z = x_a + i x_b, becomes z * exp(i phi)
    with phi = pos * theta^(-2i/d_a) (the textbook complex form, numpy complex exp)."""
    F, Hp, Wp, s0, D = 2, 3, 4, 2, 32
    dims, theta = (8, 12, 10), 100.0
    S = s0 + F * Hp * Wp + 3
    x = _rope_x(1, 2, S, D, seed=31)
    xd = _dec(x)
    for inter in (True, False):
        y = orc.rope3d(x, (F, Hp, Wp), s0, dims, theta, inter)
        for s in range(s0, s0 + F * Hp * Wp):
            g = s - s0
            pos = (g // (Hp * Wp), (g // Wp) % Hp, g % Wp)
            base = 0
            for a, da in enumerate(dims):
                for i in range(da // 2):
                    ia, ib = (base + 2 * i, base + 2 * i + 1) if inter else (base + i, base + i + da // 2)
                    z = (xd[:, :, s, ia] + 1j * xd[:, :, s, ib]) * np.exp(1j * pos[a] * theta ** (-2.0 * i / da))
                    np.testing.assert_allclose(y[:, :, s, ia], z.real, rtol=0, atol=1e-12)
                    np.testing.assert_allclose(y[:, :, s, ib], z.imag, rtol=0, atol=1e-12)
                base += da


def pin_rope_norm_and_identity(orc):
    """Rotations keep every pair's norm; the grid origin, tokens outside the grid and
    the dims past d_t + d_h + d_w are unchanged."""
    F, Hp, Wp, s0, D = 3, 2, 5, 4, 40
    dims = (10, 8, 12)
    S = s0 + F * Hp * Wp + 6
    x = _rope_x(2, 1, S, D, seed=32, gain=2.0)
    xd = _dec(x)
    y = orc.rope3d(x, (F, Hp, Wp), s0, dims, 10000.0, True)
    np.testing.assert_allclose(np.sum(y[..., :30].reshape(2, 1, S, 15, 2) ** 2, -1),
                               np.sum(xd[..., :30].reshape(2, 1, S, 15, 2) ** 2, -1), rtol=1e-13, atol=1e-13)
    np.testing.assert_array_equal(y[..., 30:], xd[..., 30:])
    outside = list(range(s0)) + list(range(s0 + F * Hp * Wp, S))
    np.testing.assert_array_equal(y[:, :, outside], xd[:, :, outside])
    np.testing.assert_array_equal(y[:, :, s0], xd[:, :, s0])          # position (0, 0, 0)


def pin_rope_one_axis_each(orc):
    """A step along t turns only the t dims, along h only the h dims, along w only the w dims."""
    F, Hp, Wp, D = 2, 2, 2, 24
    dims = (8, 8, 8)
    x = _rope_x(1, 1, F * Hp * Wp, D, seed=33)
    xd = _dec(x)
    y = orc.rope3d(x, (F, Hp, Wp), 0, dims, 50.0, False)
    for s, axis in ((4, 0), (2, 1), (1, 2)):          # (1,0,0), (0,1,0), (0,0,1)
        for a in range(3):
            sl = slice(8 * a, 8 * a + 8)
            if a == axis:
                assert np.max(np.abs(y[0, 0, s, sl] - xd[0, 0, s, sl])) > 1e-3
            else:
                np.testing.assert_array_equal(y[0, 0, s, sl], xd[0, 0, s, sl])


def pin_rope_relative_position(orc):
    """<R(p) q, R(p') k> depends on p - p' only: moving both tokens by the same step
    along any axis leaves their dot product unchanged."""
    F, Hp, Wp, D = 4, 4, 4, 48
    dims = (16, 16, 16)
    S = F * Hp * Wp
    rng = np.random.default_rng(34)
    qv = _bits_of(rng.standard_normal(D).astype(np.float32))
    kv = _bits_of(rng.standard_normal(D).astype(np.float32))
    idx = lambda t, h, w: (t * Hp + h) * Wp + w
    x = np.zeros((1, 1, S, D), dtype=np.uint16)
    pairs = [((0, 1, 2), (1, 0, 0)), ((1, 2, 3), (2, 1, 1))]   # second pair = first shifted by (1, 1, 1)
    for (pq, pk) in pairs:
        x[0, 0, idx(*pq)] = qv
        x[0, 0, idx(*pk)] = kv
    for inter in (True, False):
        y = orc.rope3d(x, (F, Hp, Wp), 0, dims, 1000.0, inter)
        d0 = y[0, 0, idx(*pairs[0][0])] @ y[0, 0, idx(*pairs[0][1])]
        d1 = y[0, 0, idx(*pairs[1][0])] @ y[0, 0, idx(*pairs[1][1])]
        assert abs(d0 - d1) <= 1e-11 * max(1.0, abs(d0)), (d0, d1)


def pin_rope_pairing_conventions(orc):
    """The half-split pairing is the interleaved one on dims permuted inside each axis
    part (interleaved 2i, 2i+1 <-> half i, i + d_a/2)."""
    F, Hp, Wp, D = 2, 3, 2, 30
    dims = (6, 10, 12)
    x = _rope_x(1, 2, F * Hp * Wp, D, seed=35)
    perm = np.arange(D)
    base = 0
    for da in dims:
        for i in range(da // 2):
            perm[base + 2 * i] = base + i
            perm[base + 2 * i + 1] = base + i + da // 2
        base += da
    yi = orc.rope3d(np.ascontiguousarray(x[..., perm]), (F, Hp, Wp), 0, dims, 77.0, True)
    yh = orc.rope3d(x, (F, Hp, Wp), 0, dims, 77.0, False)
    np.testing.assert_allclose(yi, yh[..., perm], rtol=0, atol=1e-13)


# ---- windowed 3D attention (appendix Table 4: the LTX-2.5 VAE decoder's 11^3 neighbourhood attention)

def _coords(grid):
    F, Hp, Wp = grid
    i = np.arange(F * Hp * Wp)
    return i // (Hp * Wp), (i // Wp) % Hp, i % Wp


def _window_sets(grid, window, neighbourhood):
    """[S, S] boolean: query i may attend key j.  Independent characterisations:
    neighbourhood = the in-range run of k positions whose centre is closest to p
    (brute force over every start); truncated = {j : |j - p| <= k // 2}."""
    axes = []
    for p_arr, L, kk in zip(_coords(grid), grid, window):
        if neighbourhood:
            n = min(kk, L)
            starts = np.arange(L - n + 1)
            best = starts[np.argmin(np.abs(starts[None, :] + (n - 1) / 2.0 - np.arange(L)[:, None]), axis=1)]
            lo = best[p_arr]
            ok = (p_arr[None, :] >= lo[:, None]) & (p_arr[None, :] < lo[:, None] + n)
        else:
            ok = np.abs(p_arr[None, :] - p_arr[:, None]) <= kk // 2
        axes.append(ok)
    return axes[0] & axes[1] & axes[2]


def pin_win3d_torch_masked_sdpa(orc):
    """Both border rules against torch SDPA with the window mask, fp64 (a library)."""
    grid = (3, 4, 5)
    S = 60
    q, k, v = random_qkv(2, 2, S, S, 16, seed=41, logit_gain=1.5)
    for window, nb in (((3, 3, 3), True), ((3, 3, 3), False), ((1, 3, 5), True), ((3, 1, 3), False)):
        o, lse = orc.attn_fwd_win3d(bf16_bits(q), bf16_bits(k), bf16_bits(v), 0.3, grid, window, nb)
        mask = torch.from_numpy(_window_sets(grid, window, nb))
        qd, kd, vd = q.double(), k.double(), v.double()
        want = torch.nn.functional.scaled_dot_product_attention(qd, kd, vd, attn_mask=mask, scale=0.3)
        logits = (0.3 * (qd @ kd.transpose(-1, -2))).masked_fill(~mask, -math.inf)
        np.testing.assert_allclose(o, want.numpy(), rtol=0, atol=1e-12)
        np.testing.assert_allclose(lse, torch.logsumexp(logits, -1).numpy(), rtol=1e-13, atol=1e-12)


def pin_win3d_whole_grid_is_dense(orc):
    """A window as large as the grid (neighbourhood) or twice as large (truncated) is dense attention."""
    grid = (2, 3, 4)
    q, k, v = _inputs(1, 2, 24, 24, 8, seed=42, gain=1.4)
    o, lse = orc.attn_fwd(q, k, v, 0.5)
    for window, nb in (((3, 3, 5), True), ((3, 5, 7), False)):
        ow, lw = orc.attn_fwd_win3d(q, k, v, 0.5, grid, window, nb)
        np.testing.assert_array_equal(ow, o)
        np.testing.assert_array_equal(lw, lse)


def pin_win3d_single_cell(orc):
    """A 1 x 1 x 1 window: each query sees only its own key: O = its V, LSE = scale q.k."""
    grid = (2, 2, 3)
    q, k, v = _inputs(1, 1, 12, 12, 8, seed=43)
    o, lse = orc.attn_fwd_win3d(q, k, v, 0.7, grid, (1, 1, 1), True)
    np.testing.assert_array_equal(o, _dec(v))
    np.testing.assert_allclose(lse, 0.7 * np.einsum("bhid,bhid->bhi", _dec(q), _dec(k)), rtol=1e-15, atol=1e-14)


def pin_win3d_counts_and_interior(orc):
    """Neighbourhood windows always hold prod(min(k, L)) keys; away from the
    border both rules give the same window, hence the same result."""
    grid, window = (5, 6, 7), (3, 3, 5)
    S = 210
    q, k, v = _inputs(1, 1, S, S, 8, seed=44, gain=1.2)
    on, ln, pn = orc.attn_fwd_win3d(q, k, v, 0.4, grid, window, True, probs=True)
    ot, lt = orc.attn_fwd_win3d(q, k, v, 0.4, grid, window, False)
    assert np.all(np.count_nonzero(pn[0, 0], axis=1) == 3 * 3 * 5)
    t, h, w = _coords(grid)
    inner = (t >= 1) & (t <= 3) & (h >= 1) & (h <= 4) & (w >= 2) & (w <= 4)
    assert inner.any() and (~inner).any()
    np.testing.assert_array_equal(on[0, 0, inner], ot[0, 0, inner])
    np.testing.assert_array_equal(ln[0, 0, inner], lt[0, 0, inner])
    assert np.any(on[0, 0, ~inner] != ot[0, 0, ~inner])


ALL_PINS = [pin_single_key, pin_two_keys, pin_weights_sum_to_one, pin_constant_values,
            pin_zero_logits, pin_query_permutation, pin_key_value_permutation,
            pin_value_translation, pin_varlen_is_truncation, pin_varlen_empty_and_clamped,
            pin_row_subset, pin_torch_sdpa, pin_mpmath_brute_force, pin_large_logits_stable,
            pin_segments_one_segment_is_dense, pin_segments_packed_are_independent,
            pin_segments_prefix_is_valid_count, pin_segments_torch_masked_sdpa,
            pin_rope_complex_rotation, pin_rope_norm_and_identity, pin_rope_one_axis_each,
            pin_rope_relative_position, pin_rope_pairing_conventions,
            pin_win3d_torch_masked_sdpa, pin_win3d_whole_grid_is_dense, pin_win3d_single_cell,
            pin_win3d_counts_and_interior]
