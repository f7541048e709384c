// Geometry of windowed 3D attention, for sm_103a.
//
// What it serves (vidax paper, appendix Table 4: the LTX-2.5 VAE decoder's 3D
// neighbourhood attention, an 11 x 11 x 11 window).  The S = F*Hp*Wp tokens of
// a sequence are a (t, h, w) grid in raster order; a query attends the keys
// inside its window.  Along an axis of length L with odd window size k the
// window of position p is
//     neighbourhood: [lo, min(lo + k, L) - 1], lo = clamp(p - k/2, 0, max(L - k, 0))
//                    (shifted inward at the border);
//     truncated:     [max(p - k/2, 0), min(p + k/2, L - 1)].
// Both bounds are non-decreasing in p, so the windows of a run of positions
// [p0, p1] cover exactly [lo(p0), hi(p1)].
//
// Tiles are 3-D boxes of the grid, not runs of the raster order.  A query
// tile is a brick of qbt x qbh x qbw = 128 tokens (TMA loads it through a
// 5-D tensor map (D, Wp, Hp, F, B*H) as 128 rows, w fastest); a unit is two
// bricks stacked in t.  The union of the windows of a unit's queries is then
// one box, and the unit's key tiles are a regular grid of kbt x kbh x kbw =
// 128-token boxes laid over it from its low corner: no key-tile list is
// needed, each box's origin follows from its index.  Boxes reaching past the
// union or the grid hold keys that no query of the unit attends (TMA fills
// positions outside the grid with zeros); the per-row mask removes them.
// The host chooses both box shapes to minimise the key boxes visited; the
// pattern of one t-slice of a key box (kbh x kbw bits) fits one 32-bit word.
#pragma once

#include <cstdint>

namespace vdx {

struct WinGrid {
    int F, Hp, Wp;       // grid; S = F * Hp * Wp
    int kt, kh, kw;      // odd window sizes
    int neighbourhood;   // 1: shifted inward at the border; 0: truncated
    // log2 of the query brick and key box sides (t, h, w), each triple summing to 7
    int qlt, qlh, qlw;
    int klt, klh, klw;
    int nuh, nuw;        // units along h and w (the unit index is (jt * nuh + jh) * nuw + jw)
};

__host__ __device__ __forceinline__ void axis_window(int p, int L, int k, int neighbourhood, int &lo, int &hi)
{
    if (neighbourhood) {
        const int last = L - k > 0 ? L - k : 0;
        lo = p - k / 2;
        lo = lo < 0 ? 0 : (lo > last ? last : lo);
        hi = (lo + k < L ? lo + k : L) - 1;
    } else {
        lo = p - k / 2 < 0 ? 0 : p - k / 2;
        hi = p + k / 2 < L - 1 ? p + k / 2 : L - 1;
    }
}

// Union of the windows of positions [p0, p1] (clipped to the axis) along one axis.
__host__ __device__ __forceinline__ void axis_union(int p0, int p1, int L, int k, int neighbourhood, int &lo, int &hi)
{
    int a, b;
    p1 = p1 < L - 1 ? p1 : L - 1;
    axis_window(p0, L, k, neighbourhood, lo, a);
    axis_window(p1, L, k, neighbourhood, b, hi);
}

// A unit's geometry: the origin of its first query brick and the union box
// of its queries' windows, with the key-box counts along each axis.
struct WinUnit {
    int t0, h0, w0;            // first brick's origin (the second is qbt further in t)
    int ut, uh, uw;            // union box low corner
    int nbt, nbh, nbw;         // key boxes per axis
};

__host__ __device__ __forceinline__ WinUnit win_unit(const WinGrid &g, int qp)
{
    WinUnit u;
    const int jw = qp % g.nuw;
    const int r = qp / g.nuw;
    const int jh = r % g.nuh;
    const int jt = r / g.nuh;
    u.t0 = jt << (g.qlt + 1);
    u.h0 = jh << g.qlh;
    u.w0 = jw << g.qlw;
    int hi;
    axis_union(u.t0, u.t0 + (2 << g.qlt) - 1, g.F, g.kt, g.neighbourhood, u.ut, hi);
    u.nbt = (hi - u.ut + (1 << g.klt)) >> g.klt;
    axis_union(u.h0, u.h0 + (1 << g.qlh) - 1, g.Hp, g.kh, g.neighbourhood, u.uh, hi);
    u.nbh = (hi - u.uh + (1 << g.klh)) >> g.klh;
    axis_union(u.w0, u.w0 + (1 << g.qlw) - 1, g.Wp, g.kw, g.neighbourhood, u.uw, hi);
    u.nbw = (hi - u.uw + (1 << g.klw)) >> g.klw;
    return u;
}

// Origin of key box r of a unit.
__device__ __forceinline__ void win_box(const WinGrid &g, const WinUnit &u, int r, int &t, int &h, int &w)
{
    const int iw = r % u.nbw;
    const int q = r / u.nbw;
    const int ih = q % u.nbh;
    const int it = q / u.nbh;
    t = u.ut + (it << g.klt);
    h = u.uh + (ih << g.klh);
    w = u.uw + (iw << g.klw);
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

// Bits [lo, hi] of a 32-bit word (0 <= lo <= hi < 32).
__device__ __forceinline__ uint32_t bit_range32(int lo, int hi)
{
    const int n = hi - lo + 1;
    return (n == 32 ? 0xFFFFFFFFu : ((1u << n) - 1u)) << lo;
}

// A g-bit pattern (g a power of two, 1..32) repeated across a 32-bit word.
__device__ __forceinline__ uint32_t repeat32(uint32_t pattern, int lg)
{
#pragma unroll
    for (int s = 0; s < 5; ++s)
        if (s >= lg)
            pattern |= pattern << (1 << s);
    return pattern;
}

// The window of a query at grid position (t, h, w), one axis per word: lo in
// the low 16 bits, hi in the high 16 (grid sides below 65536).  A position
// outside the grid (a ragged brick's padding row) gets empty windows.
__device__ __forceinline__ void packed_window(const WinGrid &g, int t, int h, int w, uint32_t &tw, uint32_t &hw,
                                              uint32_t &ww)
{
    if (t >= g.F || h >= g.Hp || w >= g.Wp) {
        tw = hw = ww = 1u;   // lo = 1 > hi = 0
        return;
    }
    int lo, hi;
    axis_window(t, g.F, g.kt, g.neighbourhood, lo, hi);
    tw = static_cast<uint32_t>(lo) | (static_cast<uint32_t>(hi) << 16);
    axis_window(h, g.Hp, g.kh, g.neighbourhood, lo, hi);
    hw = static_cast<uint32_t>(lo) | (static_cast<uint32_t>(hi) << 16);
    axis_window(w, g.Wp, g.kw, g.neighbourhood, lo, hi);
    ww = static_cast<uint32_t>(lo) | (static_cast<uint32_t>(hi) << 16);
}

// 128-bit mask of the keys of the key box with origin (t, h, w) inside a
// query's window (packed as above).  Key c of the box sits at
// (t + c / (kbh kbw), h + (c / kbw) % kbh, w + c % kbw).  The (h, w) pattern of
// one t-slice (kbh x kbw bits, at most 32) is the w-range repeated over the
// slice's rows and cut to the h-range; the mask repeats it over the t-slices
// and cuts it to the t-range.  A repetition is one multiplication: a pattern
// narrower than its group times a comb (a 1 at the start of every group; no
// two copies overlap, so there is no carry).  comb_w has a 1 every kbw bits,
// comb_s every kbh kbw bits.  The t-range words depend only on the row's
// window and the box's t; they are kept in tm for the last t seen (tc), which
// the caller resets whenever the row's window changes.
__device__ __forceinline__ void window_mask(const WinGrid &g, uint32_t tw, uint32_t hw, uint32_t ww, int t, int h,
                                            int w, uint32_t comb_w, uint32_t comb_s, int &tc, uint32_t (&tm)[4],
                                            uint32_t (&m)[4])
{
    if (t != tc) {
        tc = t;
        tm[0] = tm[1] = tm[2] = tm[3] = 0u;
        const int tlo = max(static_cast<int>(tw & 0xFFFFu) - t, 0);
        const int thi = min(static_cast<int>(tw >> 16) - t, (1 << g.klt) - 1);
        if (tlo <= thi)
            set_bit_range(tm, tlo << (g.klh + g.klw), ((thi + 1) << (g.klh + g.klw)) - 1);
    }
    const int hlo = max(static_cast<int>(hw & 0xFFFFu) - h, 0), hhi = min(static_cast<int>(hw >> 16) - h, (1 << g.klh) - 1);
    const int wlo = max(static_cast<int>(ww & 0xFFFFu) - w, 0), whi = min(static_cast<int>(ww >> 16) - w, (1 << g.klw) - 1);
    uint32_t word = 0u;
    if (hlo <= hhi && wlo <= whi)
        word = ((bit_range32(wlo, whi) * comb_w) & bit_range32(hlo << g.klw, ((hhi + 1) << g.klw) - 1)) * comb_s;
#pragma unroll
    for (int i = 0; i < 4; ++i)
        m[i] = tm[i] & word;
}

}  // namespace vdx
