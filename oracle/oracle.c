/*
 * Oracle: plain fp64 CPU softmax attention forward.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may link, load or
 * call this file; only the tests, the smoke check and the bench's CPU
 * baseline leg use it.  It shares no code, header, table or helper with the
 * CUDA library under paper_2609_18077_gb300/csrc.
 *
 * What it computes.  The vidax paper (arXiv 2609.18077, Sec. 2, paragraph
 * "3D RoPE, 3D VAEs, and flash attention") runs unmasked multi-head attention
 * over patchified video tokens through flash-attention kernels, whose point is
 * to avoid materialising the full query-key matrix; the flash algorithm is
 * cited there, not restated, and it reaches the plain softmax-attention result
 * up to rounding order.  So this oracle is that plain definition, written out
 * with no tiling and no online rescaling:
 *
 *     s_j   = scale * sum_d q[i,d] * k[j,d]            for j < L
 *     m     = max_j s_j
 *     l     = sum_j exp(s_j - m)
 *     o[i,:] = (sum_j exp(s_j - m) * v[j,:]) / l
 *     lse_i = m + ln(l)                                 (natural log)
 *
 * Masked text keys (appendix Table 4, the porting-bug taxonomy: attending
 * unmasked padding tokens is a bug, and invalid key blocks are skipped through
 * segment ids rather than a dense (B,H,Sq,Sk) mask) are modelled by a
 * per-batch valid key count L_b = clamp(kv_lens[b], 0, Skv); keys j >= L_b are
 * never read.  L_b = 0 gives o = 0 and lse = -inf.
 *
 * Joint text-video attention (oracle_attn_fwd_seg) generalises the valid
 * count to segment ids, the form the same appendix entry names for
 * HunyuanVideo-1.5's joint attention over video and padded text tokens: query
 * i of sample b attends exactly the keys j with kv_seg[b,j] == q_seg[b,i], and
 * the definition above runs over that key set in ascending key order.  A query
 * whose segment owns no key gets o = 0 and lse = -inf.
 *
 * Windowed 3D attention (oracle_attn_fwd_win3d): appendix Table 4 names the
 * LTX-2.5 VAE decoder's 3D neighbourhood attention with an 11 x 11 x 11
 * window.  The S = F*Hp*Wp tokens are a (t, h, w) grid in raster order and a
 * query attends exactly the keys inside its window: along each axis of
 * length L with odd window size k, the window of the query at p is
 *     neighbourhood: [lo, lo + k) with lo = clamp(p - k/2, 0, max(L - k, 0)),
 *                    cut to [0, L) (shifted inward at the border, so it
 *                    always spans min(k, L) positions);
 *     truncated:     [max(p - k/2, 0), min(p + k/2, L - 1)].
 * The definition above then runs over that key set in ascending key order.
 *
 * 3D rotary position embedding (oracle_rope3d).  Sec. 2 of the paper
 * ("3D RoPE, 3D VAEs, and flash attention") keeps each model family's own
 * 3D RoPE convention over time, height and width without stating one.  The
 * oracle is the standard rotary embedding over a 3-D grid, parameterised by
 * the conventions those families differ in: the video tokens [s0, s0 + F*Hp*Wp)
 * of a sequence sit at grid positions (t, h, w) in raster order; the first
 * d_t head dims rotate with t, the next d_h with h, the next d_w with w, the
 * rest are untouched; inside an axis part of d_a dims, pair i is (2i, 2i+1)
 * (interleaved) or (i, i + d_a/2) (half split) and turns by the angle
 * pos * theta^(-2i/d_a):
 *     (y_a, y_b) = (x_a cos(phi) - x_b sin(phi), x_a sin(phi) + x_b cos(phi)).
 * Tokens outside the grid are copied unchanged.  Output is fp64.
 *
 * Inputs are bf16 bit patterns (uint16), decoded exactly to fp64.  All
 * arithmetic is fp64.  Layout: q [B,H,Sq,D], k and v [B,H,Skv,D], contiguous.
 * Parallelism: one OpenMP loop over (b, h, query row); each row is computed
 * independently by the same sequential code.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* Exact bf16 -> fp64: a bf16 value is the top half of an IEEE binary32. */
static double bf16_to_f64(uint16_t bits)
{
    uint32_t u = (uint32_t)bits << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/*
 * Attention for one query row against L keys of one (b, h): keys 0 .. L-1,
 * or, when idx != NULL, keys idx[0], ..., idx[L-1].
 * q: D values; k, v: [Skv, D]; s: scratch of L doubles.
 * Writes o[D], *lse and, if probs != NULL, probs[r] = softmax weight of the
 * r-th attended key.
 */
static void attend_row(const uint16_t *q, const uint16_t *k, const uint16_t *v,
                       const int *idx, int L, int D, double scale, double *s,
                       double *o, double *lse, double *probs)
{
    if (L <= 0) {
        for (int d = 0; d < D; ++d)
            o[d] = 0.0;
        *lse = -INFINITY;
        return;
    }
    /* logits */
    for (int j = 0; j < L; ++j) {
        const size_t kj = (size_t)(idx ? idx[j] : j);
        double dot = 0.0;
        for (int d = 0; d < D; ++d)
            dot += bf16_to_f64(q[d]) * bf16_to_f64(k[kj * D + d]);
        s[j] = scale * dot;
    }
    /* softmax normaliser */
    double m = s[0];
    for (int j = 1; j < L; ++j)
        if (s[j] > m)
            m = s[j];
    double l = 0.0;
    for (int j = 0; j < L; ++j)
        l += exp(s[j] - m);
    /* weighted sum of values */
    for (int d = 0; d < D; ++d)
        o[d] = 0.0;
    for (int j = 0; j < L; ++j) {
        const size_t vj = (size_t)(idx ? idx[j] : j);
        double p = exp(s[j] - m) / l;
        if (probs)
            probs[j] = p;
        for (int d = 0; d < D; ++d)
            o[d] += p * bf16_to_f64(v[vj * D + d]);
    }
    *lse = m + log(l);
}

static int valid_len(const int32_t *kv_lens, int b, int Skv)
{
    if (!kv_lens)
        return Skv;
    int L = kv_lens[b];
    if (L < 0)
        L = 0;
    if (L > Skv)
        L = Skv;
    return L;
}

/*
 * Full or row-subset attention forward.
 *
 *   rows == NULL : every query row; o is [B*H, Sq, D], lse is [B*H, Sq].
 *   rows != NULL : rows is [B*H, nrows] (query indices per (b, h));
 *                  o is [B*H, nrows, D], lse is [B*H, nrows].
 *   kv_lens == NULL : all Skv keys are valid; else int32 [B].
 *   probs (optional, tiny shapes only): [B*H, nrows or Sq, Skv], zero beyond L_b.
 *
 * Returns 0, or -1 on a bad argument or a failed allocation.
 */
int oracle_attn_fwd(const uint16_t *q, const uint16_t *k, const uint16_t *v,
                    int B, int H, int Sq, int Skv, int D, double scale,
                    const int32_t *kv_lens, const int32_t *rows, int nrows,
                    double *o, double *lse, double *probs)
{
    if (!q || !k || !v || !o || !lse || B < 0 || H < 0 || Sq < 0 || Skv < 0 || D <= 0)
        return -1;
    const int nr = rows ? nrows : Sq;
    if (nr < 0)
        return -1;
    const long total = (long)B * H * nr;
    int failed = 0;

#pragma omp parallel
    {
        double *s = (double *)malloc(sizeof(double) * (size_t)(Skv > 0 ? Skv : 1));
        if (!s) {
#pragma omp atomic write
            failed = 1;
        }
#pragma omp for schedule(dynamic, 4)
        for (long t = 0; t < total; ++t) {
            if (!s)
                continue;
            const long bh = t / nr;
            const int r = (int)(t % nr);
            const int b = (int)(bh / H);
            const int i = rows ? rows[bh * nrows + r] : r;
            if (i < 0 || i >= Sq) {
#pragma omp atomic write
                failed = 1;
                continue;
            }
            const int L = valid_len(kv_lens, b, Skv);
            const uint16_t *qi = q + ((size_t)bh * Sq + i) * D;
            const uint16_t *kb = k + (size_t)bh * Skv * D;
            const uint16_t *vb = v + (size_t)bh * Skv * D;
            double *pr = probs ? probs + (size_t)t * Skv : NULL;
            if (pr)
                for (int j = 0; j < Skv; ++j)
                    pr[j] = 0.0;
            attend_row(qi, kb, vb, NULL, L, D, scale, s, o + (size_t)t * D, lse + t, pr);
        }
        free(s);
    }
    return failed ? -1 : 0;
}

/*
 * Joint attention with segment ids: query i of sample b attends the keys j
 * with kv_seg[b*Skv + j] == q_seg[b*Sq + i] (see the header).
 *
 *   q_seg: int32 [B, Sq]; kv_seg: int32 [B, Skv] (shared by the heads).
 *   rows, o, lse: as for oracle_attn_fwd.
 *   probs (optional, tiny shapes only): [B*H, nrows or Sq, Skv], zero for
 *   keys outside the row's segment.
 *
 * Returns 0, or -1 on a bad argument or a failed allocation.
 */
int oracle_attn_fwd_seg(const uint16_t *q, const uint16_t *k, const uint16_t *v,
                        int B, int H, int Sq, int Skv, int D, double scale,
                        const int32_t *q_seg, const int32_t *kv_seg,
                        const int32_t *rows, int nrows,
                        double *o, double *lse, double *probs)
{
    if (!q || !k || !v || !o || !lse || !q_seg || !kv_seg || B < 0 || H < 0 || Sq < 0 || Skv < 0 || D <= 0)
        return -1;
    const int nr = rows ? nrows : Sq;
    if (nr < 0)
        return -1;
    const long total = (long)B * H * nr;
    const size_t cap = (size_t)(Skv > 0 ? Skv : 1);
    int failed = 0;

#pragma omp parallel
    {
        double *s = (double *)malloc(sizeof(double) * cap);
        double *ps = (double *)malloc(sizeof(double) * cap);
        int *idx = (int *)malloc(sizeof(int) * cap);
        if (!s || !ps || !idx) {
#pragma omp atomic write
            failed = 1;
        }
#pragma omp for schedule(dynamic, 4)
        for (long t = 0; t < total; ++t) {
            if (!s || !ps || !idx)
                continue;
            const long bh = t / nr;
            const int r = (int)(t % nr);
            const int b = (int)(bh / H);
            const int i = rows ? rows[bh * nrows + r] : r;
            if (i < 0 || i >= Sq) {
#pragma omp atomic write
                failed = 1;
                continue;
            }
            /* the keys of this query's segment, in ascending order */
            const int32_t seg = q_seg[(size_t)b * Sq + i];
            const int32_t *kseg = kv_seg + (size_t)b * Skv;
            int n = 0;
            for (int j = 0; j < Skv; ++j)
                if (kseg[j] == seg)
                    idx[n++] = j;
            const uint16_t *qi = q + ((size_t)bh * Sq + i) * D;
            const uint16_t *kb = k + (size_t)bh * Skv * D;
            const uint16_t *vb = v + (size_t)bh * Skv * D;
            attend_row(qi, kb, vb, idx, n, D, scale, s, o + (size_t)t * D, lse + t, probs ? ps : NULL);
            if (probs) {
                double *pr = probs + (size_t)t * Skv;
                for (int j = 0; j < Skv; ++j)
                    pr[j] = 0.0;
                for (int e = 0; e < n; ++e)
                    pr[idx[e]] = ps[e];
            }
        }
        free(s);
        free(ps);
        free(idx);
    }
    return failed ? -1 : 0;
}

/* Window [lo, hi] of position p on an axis of length L, window size k (odd). */
static void axis_window(int p, int L, int k, int neighbourhood, int *lo, int *hi)
{
    if (neighbourhood) {
        int start = p - k / 2;
        const int last_start = L - k > 0 ? L - k : 0;
        if (start < 0)
            start = 0;
        if (start > last_start)
            start = last_start;
        *lo = start;
        *hi = start + k - 1 < L - 1 ? start + k - 1 : L - 1;
    } else {
        *lo = p - k / 2 > 0 ? p - k / 2 : 0;
        *hi = p + k / 2 < L - 1 ? p + k / 2 : L - 1;
    }
}

/*
 * Windowed 3D attention over the grid F x Hp x Wp (S = F*Hp*Wp tokens per
 * sequence, raster order t, h, w), window kt x kh x kw (odd sizes); see the
 * header.  rows, o, lse, probs as for oracle_attn_fwd.
 * Returns 0, or -1 on a bad argument or a failed allocation.
 */
int oracle_attn_fwd_win3d(const uint16_t *q, const uint16_t *k, const uint16_t *v,
                          int B, int H, int F, int Hp, int Wp, int D, double scale,
                          int kt, int kh, int kw, int neighbourhood,
                          const int32_t *rows, int nrows, double *o, double *lse, double *probs)
{
    if (!q || !k || !v || !o || !lse || B < 0 || H < 0 || F < 0 || Hp < 0 || Wp < 0 || D <= 0 ||
        kt < 1 || kh < 1 || kw < 1 || !(kt & kh & kw & 1))
        return -1;
    const long S_l = (long)F * Hp * Wp;
    if (S_l > 0x7fffffffL)
        return -1;
    const int S = (int)S_l;
    const int nr = rows ? nrows : S;
    if (nr < 0)
        return -1;
    const long total = (long)B * H * nr;
    const size_t cap = (size_t)(S > 0 ? S : 1);
    int failed = 0;

#pragma omp parallel
    {
        double *s = (double *)malloc(sizeof(double) * cap);
        double *ps = (double *)malloc(sizeof(double) * cap);
        int *idx = (int *)malloc(sizeof(int) * cap);
        if (!s || !ps || !idx) {
#pragma omp atomic write
            failed = 1;
        }
#pragma omp for schedule(dynamic, 4)
        for (long t = 0; t < total; ++t) {
            if (!s || !ps || !idx)
                continue;
            const long bh = t / nr;
            const int r = (int)(t % nr);
            const int i = rows ? rows[bh * nrows + r] : r;
            if (i < 0 || i >= S) {
#pragma omp atomic write
                failed = 1;
                continue;
            }
            /* the query's grid position and window on each axis */
            const int pt = i / (Hp * Wp), ph = (i / Wp) % Hp, pw = i % Wp;
            int tlo, thi, hlo, hhi, wlo, whi;
            axis_window(pt, F, kt, neighbourhood, &tlo, &thi);
            axis_window(ph, Hp, kh, neighbourhood, &hlo, &hhi);
            axis_window(pw, Wp, kw, neighbourhood, &wlo, &whi);
            /* the keys inside it, in ascending order */
            int n = 0;
            for (int tt = tlo; tt <= thi; ++tt)
                for (int hh = hlo; hh <= hhi; ++hh)
                    for (int ww = wlo; ww <= whi; ++ww)
                        idx[n++] = (tt * Hp + hh) * Wp + ww;
            const uint16_t *qi = q + ((size_t)bh * S + i) * D;
            const uint16_t *kb = k + (size_t)bh * S * D;
            const uint16_t *vb = v + (size_t)bh * S * D;
            attend_row(qi, kb, vb, idx, n, D, scale, s, o + (size_t)t * D, lse + t, probs ? ps : NULL);
            if (probs) {
                double *pr = probs + (size_t)t * S;
                for (int j = 0; j < S; ++j)
                    pr[j] = 0.0;
                for (int e = 0; e < n; ++e)
                    pr[idx[e]] = ps[e];
            }
        }
        free(s);
        free(ps);
        free(idx);
    }
    return failed ? -1 : 0;
}

/*
 * 3D rotary embedding of x [B, H, S, D] (bf16 bits) into y (fp64, same shape);
 * see the header for the parameters.  Returns 0, or -1 on a bad argument.
 */
int oracle_rope3d(const uint16_t *x, int B, int H, int S, int D, int F, int Hp, int Wp, int s0,
                  int d_t, int d_h, int d_w, double theta, int interleaved, double *y)
{
    if (!x || !y || B < 0 || H < 0 || S < 0 || D <= 0 || F < 0 || Hp < 0 || Wp < 0 || s0 < 0 ||
        d_t < 0 || d_h < 0 || d_w < 0 || (d_t | d_h | d_w) & 1 || d_t + d_h + d_w > D || !(theta > 0.0))
        return -1;
    const long rows = (long)B * H * S;
    const long grid = (long)F * Hp * Wp;
#pragma omp parallel for schedule(static)
    for (long r = 0; r < rows; ++r) {
        const long s = r % S;
        const uint16_t *xr = x + (size_t)r * D;
        double *yr = y + (size_t)r * D;
        for (int d = 0; d < D; ++d)
            yr[d] = bf16_to_f64(xr[d]);
        const long g = s - s0;
        if (g < 0 || g >= grid)
            continue;
        /* grid position of this token, raster order (t, h, w) */
        const long pos[3] = {g / ((long)Hp * Wp), (g / Wp) % Hp, g % Wp};
        const int len[3] = {d_t, d_h, d_w};
        int base = 0;
        for (int a = 0; a < 3; ++a) {
            const int da = len[a];
            for (int i = 0; i < da / 2; ++i) {
                const double phi = (double)pos[a] * pow(theta, -2.0 * i / da);
                const int ia = base + (interleaved ? 2 * i : i);
                const int ib = base + (interleaved ? 2 * i + 1 : i + da / 2);
                const double xa = bf16_to_f64(xr[ia]), xb = bf16_to_f64(xr[ib]);
                yr[ia] = xa * cos(phi) - xb * sin(phi);
                yr[ib] = xa * sin(phi) + xb * cos(phi);
            }
            base += da;
        }
    }
    return 0;
}

/* Threads the OpenMP loop may use (n <= 0 keeps the runtime default). */
int oracle_set_threads(int n)
{
#ifdef _OPENMP
    if (n > 0)
        omp_set_num_threads(n);
    return omp_get_max_threads();
#else
    (void)n;
    return 1;
#endif
}
