// Host-side check of the windowed-attention geometry in csrc/window_tiles.cuh,
// compiled with a plain C++ compiler (the CUDA qualifiers defined away), so
// the functions the kernel runs are the ones checked.  For every brick and
// key-box shape the kernel may use (each side a power of two, 128 tokens,
// a t-slice of at most 32 keys), over grids with ragged sides, windows larger
// than the grid and both border rules, it checks against brute force:
//   1. coverage: every key in the window of every in-grid query of a unit
//      lies inside one of the unit's key boxes (so no attended key is
//      skipped);
//   2. masks: window_mask, driven as the kernel drives it (combs, the
//      t-range cache reset at each unit, boxes in index order), sets exactly
//      the bits of the box's keys inside the row's window;
//   3. a brick row outside the grid gets an all-zero mask in every box.
// Prints "ok <cases>" and exits 0, or prints the first mismatch and exits 1.
#include <algorithm>
#include <climits>
#include <cstdint>
#include <cstdio>
#include <cstdlib>

using std::max;
using std::min;
#define __host__
#define __device__
#define __forceinline__ inline
#include "../paper_2609_18077_gb300/csrc/window_tiles.cuh"

namespace {

struct Case {
    int F, Hp, Wp, kt, kh, kw;
};

long long g_cases = 0;

// Checks one grid, window, border rule and shape pair on the units listed
// (every unit when stride == 1).  Returns false on the first mismatch.
bool check(const Case &c, int nb, int qlt, int qlh, int qlw, int klt, int klh, int klw, int stride)
{
    vdx::WinGrid g{};
    g.F = c.F, g.Hp = c.Hp, g.Wp = c.Wp;
    g.kt = c.kt, g.kh = c.kh, g.kw = c.kw;
    g.neighbourhood = nb;
    g.qlt = qlt, g.qlh = qlh, g.qlw = qlw;
    g.klt = klt, g.klh = klh, g.klw = klw;
    const int nut = (c.F + (2 << qlt) - 1) / (2 << qlt);
    g.nuh = (c.Hp + (1 << qlh) - 1) >> qlh;
    g.nuw = (c.Wp + (1 << qlw) - 1) >> qlw;
    const int units = nut * g.nuh * g.nuw;
    const uint32_t comb_w = vdx::repeat32(1u, klw), comb_s = vdx::repeat32(1u, klh + klw);
    const int kbt = 1 << klt, kbh = 1 << klh, kbw = 1 << klw;
    for (int qp = 0; qp < units; qp += stride) {
        const vdx::WinUnit u = vdx::win_unit(g, qp);
        const int nbox = u.nbt * u.nbh * u.nbw;
        static int origin[4096][3];   // box origins of the unit (at most 32 x 32 x 4 boxes here)
        if (nbox > 4096) {
            std::printf("too many boxes: %d\n", nbox);
            return false;
        }
        for (int r = 0; r < nbox; ++r)
            vdx::win_box(g, u, r, origin[r][0], origin[r][1], origin[r][2]);
        for (int t = 0; t < 2; ++t)
            for (int row = 0; row < 128; ++row) {
                // the kernel's row position (w fastest, then h, then t)
                const int pw = u.w0 + (row & ((1 << qlw) - 1));
                const int ph = u.h0 + ((row >> qlw) & ((1 << qlh) - 1));
                const int pt = u.t0 + (t << qlt) + (row >> (qlw + qlh));
                const bool on = pt < c.F && ph < c.Hp && pw < c.Wp;
                uint32_t tw, hw, ww;
                vdx::packed_window(g, pt, ph, pw, tw, hw, ww);
                int tlo = 1, thi = 0, hlo = 1, hhi = 0, wlo = 1, whi = 0;   // the row's window (empty off the grid)
                if (on) {
                    vdx::axis_window(pt, c.F, c.kt, nb, tlo, thi);
                    vdx::axis_window(ph, c.Hp, c.kh, nb, hlo, hhi);
                    vdx::axis_window(pw, c.Wp, c.kw, nb, wlo, whi);
                    // 1. coverage of the row's window by the unit's boxes
                    if (tlo < u.ut || thi >= u.ut + u.nbt * kbt || hlo < u.uh || hhi >= u.uh + u.nbh * kbh ||
                        wlo < u.uw || whi >= u.uw + u.nbw * kbw) {
                        std::printf("coverage: grid %d %d %d win %d %d %d nb %d bricks %d %d %d boxes %d %d %d unit %d "
                                    "row %d\n",
                                    c.F, c.Hp, c.Wp, c.kt, c.kh, c.kw, nb, qlt, qlh, qlw, klt, klh, klw, qp, row);
                        return false;
                    }
                }
                // 2 and 3. masks, with the kernel's cache protocol
                int tc = INT_MIN;
                uint32_t tm[4] = {0u, 0u, 0u, 0u};
                for (int r = 0; r < nbox; ++r) {
                    const int bt = origin[r][0], bh = origin[r][1], bw = origin[r][2];
                    uint32_t m[4];
                    vdx::window_mask(g, tw, hw, ww, bt, bh, bw, comb_w, comb_s, tc, tm, m);
                    for (int k = 0; k < 128; ++k) {
                        const int kt = bt + (k >> (klh + klw)), kh = bh + ((k >> klw) & (kbh - 1)), kw = bw + (k & (kbw - 1));
                        const bool want = kt >= tlo && kt <= thi && kh >= hlo && kh <= hhi && kw >= wlo && kw <= whi;
                        const bool got = (m[k >> 5] >> (k & 31)) & 1u;
                        if (want != got) {
                            std::printf("mask: grid %d %d %d win %d %d %d nb %d bricks %d %d %d boxes %d %d %d unit %d "
                                        "row %d box %d key %d: want %d got %d\n",
                                        c.F, c.Hp, c.Wp, c.kt, c.kh, c.kw, nb, qlt, qlh, qlw, klt, klh, klw, qp, row, r, k,
                                        int(want), int(got));
                            return false;
                        }
                    }
                }
            }
    }
    ++g_cases;
    return true;
}

}  // namespace

int main()
{
    // Grids of a few hundred tokens: windows larger than the grid, axes of
    // length 1 and a single token.  Each border rule takes a rotating fifth
    // of the 756 shape pairs, so every brick shape and every box shape is
    // checked many times under each rule.
    const Case tiny[] = {{4, 6, 9, 3, 3, 3}, {2, 3, 4, 3, 5, 7}, {3, 5, 7, 1, 1, 1}, {7, 1, 30, 3, 1, 5},
                         {1, 1, 1, 1, 1, 1}, {3, 2, 5, 9, 9, 9}, {2, 9, 13, 1, 7, 5}};
    for (int nb = 0; nb < 2; ++nb) {
        int pair = 0;
        for (int qlt = 0; qlt <= 7; ++qlt)
            for (int qlh = 0; qlt + qlh <= 7; ++qlh)
                for (int klt = 2; klt <= 7; ++klt)
                    for (int klh = 0; klt + klh <= 7; ++klh, ++pair) {
                        if ((pair + qlt + 2 * nb) % 5 != 0)
                            continue;
                        for (const Case &c : tiny)
                            if (!check(c, nb, qlt, qlh, 7 - qlt - qlh, klt, klh, 7 - klt - klh, 1))
                                return 1;
                    }
    }
    // Larger grids (the other windowed GPU test grids, the decoder's 11^3
    // window on a small480-sized grid, the win3d workload's grid): a spread of
    // shape pairs, every sixth (large grids: fourteenth) unit.
    const Case mid[] = {{3, 8, 50, 3, 5, 11}, {9, 17, 23, 5, 3, 7}, {5, 4, 300, 1, 3, 21}, {6, 12, 20, 5, 5, 5},
                        {8, 16, 24, 7, 3, 5}};
    const Case large[] = {{16, 32, 48, 11, 11, 11}, {21, 30, 52, 11, 11, 11}};
    const int shapes[][6] = {{3, 3, 1, 4, 1, 2}, {2, 3, 2, 3, 2, 2}, {3, 2, 2, 4, 2, 1}, {1, 3, 3, 2, 2, 3},
                             {0, 0, 7, 2, 0, 5}, {7, 0, 0, 7, 0, 0}, {0, 7, 0, 2, 5, 0}, {2, 2, 3, 5, 1, 1}};
    for (int nb = 0; nb < 2; ++nb)
        for (const auto &sh : shapes) {
            for (const Case &c : mid)
                if (!check(c, nb, sh[0], sh[1], sh[2], sh[3], sh[4], sh[5], 6))
                    return 1;
            for (const Case &c : large)
                if (!check(c, nb, sh[0], sh[1], sh[2], sh[3], sh[4], sh[5], 14))
                    return 1;
        }
    std::printf("ok %lld\n", g_cases);
    return 0;
}
