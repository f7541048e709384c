// Key-tile lists of joint attention with segment ids, for sm_103a.
//
// What it serves (vidax paper, appendix Table 4): HunyuanVideo-1.5's joint
// attention over video and padded text tokens keeps its O(S) memory only
// when padding is masked through segment ids that let the kernel skip key
// blocks no query of a block may attend, instead of a dense (B, H, Sq, Sk)
// mask.  Query i of sample b attends key j iff q_seg[b, i] == kv_seg[b, j].
//
// Two small launches ahead of the attention kernel build, for every
// (sample, pair of 128-row query tiles) -- the attention kernel's work unit,
// shared by all heads -- the ordered list of key tiles it must visit:
//   1. seg_tile_ranges_kernel: (min, max) segment id of every 128-key tile
//      and every 128-row query tile (one warp per tile);
//   2. seg_tile_lists_kernel: one warp per (sample, query-tile pair) keeps
//      the key tiles whose id range meets either query tile's range, in
//      ascending order, and marks per query tile whether the tile needs the
//      element-wise id comparison (it does unless the query tile and the key
//      tile each hold a single id, the same one).
// A range test can keep a tile that holds no matching key (ids interleaved);
// the element-wise comparison then masks all of it, so the result is exact
// either way and only the skipped work depends on the id layout.
#pragma once

#include <climits>
#include <cstdint>

namespace vdx {

// List entry: key tile index in the low 30 bits; bit 30 + t set when query
// tile t of the unit must compare ids element by element on this key tile.
constexpr uint32_t SEG_TILE_BITS = 0x3FFFFFFFu;
constexpr int SEG_MASK_SHIFT = 30;

// One warp per tile: tiles [0, B * n_kt) are key tiles, then B * n_qt query
// tiles.  An empty range (no element) is (INT_MAX, INT_MIN).
__global__ void __launch_bounds__(256) seg_tile_ranges_kernel(const int *__restrict__ q_seg,
                                                              const int *__restrict__ kv_seg, int B, int Sq, int Skv,
                                                              int n_qt, int n_kt, int2 *__restrict__ qrange,
                                                              int2 *__restrict__ krange)
{
    const long long w = (static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    const long long nk = static_cast<long long>(B) * n_kt;
    const long long nq = static_cast<long long>(B) * n_qt;
    if (w >= nk + nq)
        return;
    const bool key = w < nk;
    const long long idx = key ? w : w - nk;
    const int per = key ? n_kt : n_qt;
    const int b = static_cast<int>(idx / per);
    const int tile = static_cast<int>(idx - static_cast<long long>(b) * per);
    const int S = key ? Skv : Sq;
    const int *seg = (key ? kv_seg : q_seg) + static_cast<size_t>(b) * S;
    int lo = INT_MAX, hi = INT_MIN;
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const int c = tile * 128 + e * 32 + lane;
        if (c < S) {
            const int x = __ldg(seg + c);
            lo = min(lo, x);
            hi = max(hi, x);
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        lo = min(lo, __shfl_xor_sync(0xFFFFFFFFu, lo, o));
        hi = max(hi, __shfl_xor_sync(0xFFFFFFFFu, hi, o));
    }
    if (lane == 0)
        (key ? krange : qrange)[idx] = make_int2(lo, hi);
}

// One warp per (sample b, query-tile pair qp): tlist[(b * q_pairs + qp) * n_kt + r]
// for r < tcount[b * q_pairs + qp].
__global__ void __launch_bounds__(256) seg_tile_lists_kernel(const int2 *__restrict__ qrange,
                                                             const int2 *__restrict__ krange, int B, int q_pairs,
                                                             int n_qt, int n_kt, uint32_t *__restrict__ tlist,
                                                             int *__restrict__ tcount)
{
    const long long w = (static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (w >= static_cast<long long>(B) * q_pairs)
        return;
    const int b = static_cast<int>(w / q_pairs);
    const int qp = static_cast<int>(w - static_cast<long long>(b) * q_pairs);
    const int2 q0 = qrange[static_cast<size_t>(b) * n_qt + 2 * qp];
    const int2 q1 = 2 * qp + 1 < n_qt ? qrange[static_cast<size_t>(b) * n_qt + 2 * qp + 1] : make_int2(INT_MAX, INT_MIN);
    const int2 *kr_b = krange + static_cast<size_t>(b) * n_kt;
    uint32_t *out = tlist + static_cast<size_t>(w) * n_kt;
    int n = 0;
    for (int base = 0; base < n_kt; base += 32) {
        const int j = base + lane;
        bool keep = false;
        uint32_t e = 0;
        if (j < n_kt) {
            const int2 kr = kr_b[j];
            const bool meets0 = kr.y >= q0.x && kr.x <= q0.y;
            const bool meets1 = kr.y >= q1.x && kr.x <= q1.y;
            keep = meets0 || meets1;
            const bool one_id = kr.x == kr.y;
            const bool same0 = one_id && q0.x == q0.y && q0.x == kr.x;
            const bool same1 = one_id && q1.x == q1.y && q1.x == kr.x;
            e = static_cast<uint32_t>(j) | (same0 ? 0u : 1u << SEG_MASK_SHIFT) |
                (same1 ? 0u : 1u << (SEG_MASK_SHIFT + 1));
        }
        const unsigned kept = __ballot_sync(0xFFFFFFFFu, keep);
        if (keep)
            out[n + __popc(kept & ((1u << lane) - 1u))] = e;
        n += __popc(kept);
    }
    if (lane == 0)
        tcount[w] = n;
}

}  // namespace vdx
