// 3D rotary position embedding over a (t, h, w) token grid, for sm_103a.
//
// What it computes (vidax paper, Sec. 2 "3D RoPE, 3D VAEs, and flash
// attention": each model family keeps its own 3D RoPE convention over time,
// height and width).  The standard rotary embedding, parameterised by what the
// conventions differ in: tokens [s0, s0 + F*Hp*Wp) of every sequence sit at
// grid positions (t, h, w) in raster order; head dims [0, d_t) turn with t,
// [d_t, d_t + d_h) with h, the next d_w with w, the rest are copied.  Inside
// an axis part of d_a dims, pair i is (2i, 2i+1) (interleaved) or
// (i, i + d_a/2) (half split) and turns by pos * theta^(-2i/d_a):
//     (y_a, y_b) = (x_a cos phi - x_b sin phi, x_a sin phi + x_b cos phi).
// Tokens outside the grid are copied.  Arithmetic in fp32, output rounded to
// bf16 (nearest even).
//
// Memory-bound elementwise work (one read and one write of x): a thread owns
// one pair (or, interleaved with D a multiple of 8, four consecutive pairs =
// 16 bytes) of one token, computes the angles once and applies them to the
// token's row in every (b, h), six rows in flight at a time, so a block
// reads whole rows (consecutive tokens are consecutive rows) and the sine and
// cosine cost is shared by the B*H rows.
#pragma once

#include <cuda_bf16.h>
#include <cstdint>

namespace vdx {

struct RopeParams {
    const __nv_bfloat16 *x;
    __nv_bfloat16 *y;       // may equal x (in place)
    int BH, S, D;
    int F, Hp, Wp, s0;
    int d_t, d_h, d_w;
    float log2_theta;
    int copy_all;           // y != x: also write the untouched pairs and tokens
};

// Axis part of rotated pair `pair` (< (d_t + d_h + d_w) / 2): its axis a
// (0 t, 1 h, 2 w), its index i inside the part, the part's width da and first
// dim base.
__device__ __forceinline__ void pair_axis(const RopeParams &p, int pair, int &a, int &i, int &da, int &base)
{
    a = 0;
    base = 0;
    da = p.d_t;
    i = pair;
    if (i >= p.d_t / 2) {
        i -= p.d_t / 2;
        base = p.d_t;
        da = p.d_h;
        a = 1;
        if (i >= p.d_h / 2) {
            i -= p.d_h / 2;
            base += p.d_h;
            da = p.d_w;
            a = 2;
        }
    }
}

// theta^(-2i/da) as 2^(-2i/da * log2 theta).
__device__ __forceinline__ float pair_inv_freq(int i, int da, float log2_theta)
{
    return exp2f(-2.f * static_cast<float>(i) / static_cast<float>(da) * log2_theta);
}

// Cosine and sine of pos * inv_freq.  The angle is reduced to [-pi, pi]
// (Cody and Waite: 2 pi = 6.28125, exact in few bits, plus a small
// remainder, so k * 6.28125 is exact), then the fast sine and cosine, whose
// documented error on that interval is 2^-21.4.
__device__ __forceinline__ void turn_angle(int pos, float inv_freq, float &c, float &sn)
{
    float ph = static_cast<float>(pos) * inv_freq;
    const float k = rintf(ph * 0.15915494309189535f);
    ph = fmaf(-k, 6.28125f, ph);
    ph = fmaf(-k, 1.9353071795864769253e-3f, ph);
    __sincosf(ph, &sn, &c);
}

// Pair `pair` of a row: its two element indices, and whether and how far it turns
// for grid offset g (g outside [0, F*Hp*Wp): no turn).
template <bool INTER>
__device__ __forceinline__ bool pair_turn(const RopeParams &p, int pair, long long g, bool on_grid, int &ia, int &ib,
                                          float &c, float &sn)
{
    const int rot = (p.d_t + p.d_h + p.d_w) / 2;   // rotated pairs
    c = 1.f;
    sn = 0.f;
    if (pair >= rot) {
        // dims past the rotated parts: copied in adjacent pairs
        ia = 2 * pair;
        ib = ia + 1;
        return false;
    }
    int a, i, da, base;
    pair_axis(p, pair, a, i, da, base);
    ia = base + (INTER ? 2 * i : i);
    ib = base + (INTER ? 2 * i + 1 : i + da / 2);
    if (!on_grid)
        return false;
    const long long hw = static_cast<long long>(p.Hp) * p.Wp;
    const int pos = a == 0 ? static_cast<int>(g / hw)
                           : (a == 1 ? static_cast<int>((g / p.Wp) % p.Hp) : static_cast<int>(g % p.Wp));
    turn_angle(pos, pair_inv_freq(i, da, p.log2_theta), c, sn);
    return true;
}

// One adjacent bf16 pair (x_a in the low half) turned by (c, sn).  Rounded
// products and a fused add, spelled out so that the vectorised kernel and the
// one-pair-per-thread kernel give the same bits.
__device__ __forceinline__ uint32_t rotate_pair(uint32_t word, float c, float sn)
{
    const __nv_bfloat162 e = *reinterpret_cast<const __nv_bfloat162 *>(&word);
    const float xa = __low2float(e), xb = __high2float(e);
    const __nv_bfloat162 o = __floats2bfloat162_rn(__fmaf_rn(xa, c, __fmul_rn(-xb, sn)),
                                                   __fmaf_rn(xa, sn, __fmul_rn(xb, c)));
    return *reinterpret_cast<const uint32_t *>(&o);
}

constexpr int ROPE_ROWS = 6;   // (b, h) rows loaded before any is stored

// Interleaved pairing, D a multiple of 8: one token's 16-byte chunk q4 (four
// consecutive pairs) in every (b, h) row.
__device__ __forceinline__ void rope3d_vec_token(const RopeParams &p, int q4, int s)
{
    const long long g = static_cast<long long>(s) - p.s0;
    const bool on_grid = g >= 0 && g < static_cast<long long>(p.F) * p.Hp * p.Wp;
    float c[4], sn[4];
    bool turn[4], any = false;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        int ia, ib;
        turn[k] = pair_turn<true>(p, 4 * q4 + k, g, on_grid, ia, ib, c[k], sn[k]);
        any |= turn[k];
    }
    if (!any && !p.copy_all)
        return;
    const size_t row_stride = static_cast<size_t>(p.S) * p.D;
    const size_t off = static_cast<size_t>(s) * p.D + 8 * q4;
    for (int bh0 = 0; bh0 < p.BH; bh0 += ROPE_ROWS) {
        uint4 v[ROPE_ROWS];
#pragma unroll
        for (int r = 0; r < ROPE_ROWS; ++r)
            if (bh0 + r < p.BH)
                v[r] = *reinterpret_cast<const uint4 *>(p.x + static_cast<size_t>(bh0 + r) * row_stride + off);
#pragma unroll
        for (int r = 0; r < ROPE_ROWS; ++r) {
            if (bh0 + r >= p.BH)
                break;
            uint32_t w[4] = {v[r].x, v[r].y, v[r].z, v[r].w};
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                if (!turn[k])
                    continue;   // copied bit for bit
                w[k] = rotate_pair(w[k], c[k], sn[k]);
            }
            *reinterpret_cast<uint4 *>(p.y + static_cast<size_t>(bh0 + r) * row_stride + off) =
                make_uint4(w[0], w[1], w[2], w[3]);
        }
    }
}

// Block: (D/8) x TOK tokens; the grid (a multiple of the SM count, so that
// every SM gets the same share) strides over the tokens.
constexpr int ROPE_VEC_BLOCKS_PER_SM = 4;   // residency the grid is sized for

__global__ void __launch_bounds__(256, ROPE_VEC_BLOCKS_PER_SM) rope3d_vec_kernel(const RopeParams p)
{
    for (int s = blockIdx.x * blockDim.y + threadIdx.y; s < p.S; s += gridDim.x * blockDim.y)
        rope3d_vec_token(p, threadIdx.x, s);
}

// Any pairing and even D: a thread owns one pair of a token.  Block: (D/2) x
// TOK tokens, grid ceil(S / TOK).
template <bool INTER>
__global__ void __launch_bounds__(256) rope3d_kernel(const RopeParams p)
{
    const int pair = threadIdx.x;
    const int s = blockIdx.x * blockDim.y + threadIdx.y;
    if (s >= p.S)
        return;
    const long long g = static_cast<long long>(s) - p.s0;
    const bool on_grid = g >= 0 && g < static_cast<long long>(p.F) * p.Hp * p.Wp;
    int ia, ib;
    float c, sn;
    const bool turns = pair_turn<INTER>(p, pair, g, on_grid, ia, ib, c, sn);
    if (!turns && !p.copy_all)
        return;
    const bool packed = INTER || pair >= (p.d_t + p.d_h + p.d_w) / 2;   // elements ia, ia + 1
    const size_t row_stride = static_cast<size_t>(p.S) * p.D;
    const size_t off = static_cast<size_t>(s) * p.D;
    for (int bh0 = 0; bh0 < p.BH; bh0 += ROPE_ROWS) {
        float xa[ROPE_ROWS], xb[ROPE_ROWS];
#pragma unroll
        for (int r = 0; r < ROPE_ROWS; ++r) {
            if (bh0 + r >= p.BH)
                break;
            const size_t o = static_cast<size_t>(bh0 + r) * row_stride + off;
            if (packed) {
                const __nv_bfloat162 v = *reinterpret_cast<const __nv_bfloat162 *>(p.x + o + ia);
                xa[r] = __low2float(v);
                xb[r] = __high2float(v);
            } else {
                xa[r] = __bfloat162float(p.x[o + ia]);
                xb[r] = __bfloat162float(p.x[o + ib]);
            }
        }
#pragma unroll
        for (int r = 0; r < ROPE_ROWS; ++r) {
            if (bh0 + r >= p.BH)
                break;
            const size_t o = static_cast<size_t>(bh0 + r) * row_stride + off;
            // bf16 -> fp32 -> bf16 is an exact copy; turned pairs as in rotate_pair
            const float ya = turns ? __fmaf_rn(xa[r], c, __fmul_rn(-xb[r], sn)) : xa[r];
            const float yb = turns ? __fmaf_rn(xa[r], sn, __fmul_rn(xb[r], c)) : xb[r];
            if (packed) {
                *reinterpret_cast<__nv_bfloat162 *>(p.y + o + ia) = __floats2bfloat162_rn(ya, yb);
            } else {
                p.y[o + ia] = __float2bfloat16_rn(ya);
                p.y[o + ib] = __float2bfloat16_rn(yb);
            }
        }
    }
}

}  // namespace vdx
