// Key-tile lists of windowed 3D attention, for sm_103a.
//
// What it serves (vidax paper, appendix Table 4: the LTX-2.5 VAE decoder's 3D
// neighbourhood attention, an 11 x 11 x 11 window).  The S = F*Hp*Wp tokens of
// a sequence are a (t, h, w) grid in raster order; a query attends the keys
// inside its window.  Along an axis of length L with odd window size k the
// window of position p is
//     neighbourhood: [lo, min(lo + k, L) - 1], lo = clamp(p - k/2, 0, max(L - k, 0))
//                    (shifted inward at the border);
//     truncated:     [max(p - k/2, 0), min(p + k/2, L - 1)].
// Both bounds are non-decreasing in p.
//
// One small launch before the attention kernel builds, for every pair of
// 128-row query tiles (the attention kernel's unit; the same for every batch
// and head), the ordered list of key tiles holding at least one key inside
// the unit's window box -- per axis, the union of the windows of the unit's
// smallest and largest coordinate, a superset of every query's window -- and
// marks per query tile whether the key tile needs the element-wise window
// test (it does not when all its keys lie inside the intersection of that
// query tile's windows).
#pragma once

#include <climits>
#include <cstdint>

#include "segment_tiles.cuh"

namespace vdx {

struct WinGrid {
    int F, Hp, Wp;       // grid; S = F * Hp * Wp
    int kt, kh, kw;      // odd window sizes
    int neighbourhood;   // 1: shifted inward at the border; 0: truncated
};

__device__ __forceinline__ void axis_window(int p, int L, int k, int neighbourhood, int &lo, int &hi)
{
    if (neighbourhood) {
        const int last = L - k > 0 ? L - k : 0;
        lo = min(max(p - k / 2, 0), last);
        hi = min(lo + k, L) - 1;
    } else {
        lo = max(p - k / 2, 0);
        hi = min(p + k / 2, L - 1);
    }
}

// Coordinates of token index i.
__device__ __forceinline__ void grid_pos(const WinGrid &g, int i, int &t, int &h, int &w)
{
    const int hw = g.Hp * g.Wp;
    t = i / hw;
    const int r = i - t * hw;
    h = r / g.Wp;
    w = r - h * g.Wp;
}

// One warp per query-tile pair qp: tlist[qp * n_kt + r] for r < tcount[qp].
__global__ void __launch_bounds__(256) win_tile_lists_kernel(const WinGrid g, int S, int q_pairs, int n_kt,
                                                             uint32_t *__restrict__ tlist, int *__restrict__ tcount)
{
    const int qp = static_cast<int>((static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5);
    const int lane = threadIdx.x & 31;
    if (qp >= q_pairs)
        return;
    // per query tile t: the smallest and largest t, h, w among its rows
    int mn[2][3], mx[2][3];
#pragma unroll
    for (int q = 0; q < 2; ++q) {
#pragma unroll
        for (int a = 0; a < 3; ++a) {
            mn[q][a] = INT_MAX;
            mx[q][a] = INT_MIN;
        }
        for (int e = lane; e < 128; e += 32) {
            const int i = (2 * qp + q) * 128 + e;
            if (i < S) {
                int c[3];
                grid_pos(g, i, c[0], c[1], c[2]);
#pragma unroll
                for (int a = 0; a < 3; ++a) {
                    mn[q][a] = min(mn[q][a], c[a]);
                    mx[q][a] = max(mx[q][a], c[a]);
                }
            }
        }
#pragma unroll
        for (int a = 0; a < 3; ++a)
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                mn[q][a] = min(mn[q][a], __shfl_xor_sync(0xFFFFFFFFu, mn[q][a], o));
                mx[q][a] = max(mx[q][a], __shfl_xor_sync(0xFFFFFFFFu, mx[q][a], o));
            }
    }
    const int len[3] = {g.F, g.Hp, g.Wp};
    const int ks[3] = {g.kt, g.kh, g.kw};
    // union box of both tiles and, per tile, the intersection of its windows
    int ulo[3], uhi[3], ilo[2][3], ihi[2][3];
    bool has[2];
#pragma unroll
    for (int q = 0; q < 2; ++q)
        has[q] = mn[q][0] != INT_MAX;
#pragma unroll
    for (int a = 0; a < 3; ++a) {
        ulo[a] = INT_MAX;
        uhi[a] = INT_MIN;
#pragma unroll
        for (int q = 0; q < 2; ++q) {
            ilo[q][a] = 0;
            ihi[q][a] = -1;
            if (!has[q])
                continue;
            int lo0, hi0, lo1, hi1;
            axis_window(mn[q][a], len[a], ks[a], g.neighbourhood, lo0, hi0);
            axis_window(mx[q][a], len[a], ks[a], g.neighbourhood, lo1, hi1);
            ulo[a] = min(ulo[a], lo0);
            uhi[a] = max(uhi[a], hi1);
            ilo[q][a] = lo1;      // bounds are monotone: the largest lo and the smallest hi
            ihi[q][a] = hi0;
        }
    }
    uint32_t *out = tlist + static_cast<size_t>(qp) * n_kt;
    int n = 0;
    for (int j = 0; j < n_kt; ++j) {
        // does any of the tile's keys lie in the union box / in each intersection box?
        bool any = false, all0 = true, all1 = true;
        for (int e = lane; e < 128; e += 32) {
            const int i = j * 128 + e;
            if (i >= S)
                continue;
            int c[3];
            grid_pos(g, i, c[0], c[1], c[2]);
            bool in_u = true, in0 = true, in1 = true;
#pragma unroll
            for (int a = 0; a < 3; ++a) {
                in_u &= c[a] >= ulo[a] && c[a] <= uhi[a];
                in0 &= c[a] >= ilo[0][a] && c[a] <= ihi[0][a];
                in1 &= c[a] >= ilo[1][a] && c[a] <= ihi[1][a];
            }
            any |= in_u;
            all0 &= in0;
            all1 &= in1;
        }
        any = __any_sync(0xFFFFFFFFu, any);
        all0 = __all_sync(0xFFFFFFFFu, all0) && has[0];
        all1 = __all_sync(0xFFFFFFFFu, all1) && has[1];
        if (any) {
            if (lane == 0)
                out[n] = static_cast<uint32_t>(j) | (all0 ? 0u : 1u << SEG_MASK_SHIFT) |
                         (all1 ? 0u : 1u << (SEG_MASK_SHIFT + 1));
            ++n;
        }
    }
    if (lane == 0)
        tcount[qp] = n;
}

// Bits [lo, hi] (0 <= lo <= hi < 128) set in the 128-bit mask m.
__device__ __forceinline__ void set_bit_range(uint32_t (&m)[4], int lo, int hi)
{
#pragma unroll
    for (int wi = 0; wi < 4; ++wi) {
        const int a = max(lo, 32 * wi), b = min(hi, 32 * wi + 31);
        if (a <= b) {
            const int n = b - a + 1;
            const uint32_t bits = n == 32 ? 0xFFFFFFFFu : ((1u << n) - 1u);
            m[wi] |= bits << (a - 32 * wi);
        }
    }
}

// The window of query token q, one axis per word: lo in the low 16 bits, hi in
// the high 16 (grid sides below 65536).
__device__ __forceinline__ void packed_window(const WinGrid &g, int q, uint32_t &tw, uint32_t &hw, uint32_t &ww)
{
    int qt, qh, qw, lo, hi;
    grid_pos(g, q, qt, qh, qw);
    axis_window(qt, g.F, g.kt, g.neighbourhood, lo, hi);
    tw = static_cast<uint32_t>(lo) | (static_cast<uint32_t>(hi) << 16);
    axis_window(qh, g.Hp, g.kh, g.neighbourhood, lo, hi);
    hw = static_cast<uint32_t>(lo) | (static_cast<uint32_t>(hi) << 16);
    axis_window(qw, g.Wp, g.kw, g.neighbourhood, lo, hi);
    ww = static_cast<uint32_t>(lo) | (static_cast<uint32_t>(hi) << 16);
}

// 128-bit mask of the keys of key tile kt inside a query's window (packed as
// above), given the grid position (t, h, w) of the tile's first key: the
// tile's keys run through (t, h) rows of the grid; per row, the keys whose w
// lies inside the window form one range.
__device__ __forceinline__ void window_mask(const WinGrid &g, int S, uint32_t tw, uint32_t hw, uint32_t ww, int kt,
                                            int t, int h, int w, uint32_t (&m)[4])
{
    m[0] = m[1] = m[2] = m[3] = 0u;
    const int tlo = static_cast<int>(tw & 0xFFFFu), thi = static_cast<int>(tw >> 16);
    const int hlo = static_cast<int>(hw & 0xFFFFu), hhi = static_cast<int>(hw >> 16);
    const int wlo = static_cast<int>(ww & 0xFFFFu), whi = static_cast<int>(ww >> 16);
    const int kn = min(128, S - kt * 128);
    for (int c = 0; c < kn;) {
        const int len = min(g.Wp - w, kn - c);
        if (t >= tlo && t <= thi && h >= hlo && h <= hhi) {
            const int a = max(w, wlo), b = min(w + len - 1, whi);
            if (a <= b)
                set_bit_range(m, c + (a - w), c + (b - w));
        }
        c += len;
        w = 0;
        if (++h == g.Hp) {
            h = 0;
            ++t;
        }
    }
}

}  // namespace vdx
