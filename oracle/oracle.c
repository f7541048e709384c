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
 * Attention for one query row against the first L keys of one (b, h).
 * q: D values; k, v: [L or more, D]; s: scratch of L doubles.
 * Writes o[D], *lse and, if probs != NULL, probs[j] = softmax weight of key j.
 */
static void attend_row(const uint16_t *q, const uint16_t *k, const uint16_t *v,
                       int L, int D, double scale, double *s,
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
        double dot = 0.0;
        for (int d = 0; d < D; ++d)
            dot += bf16_to_f64(q[d]) * bf16_to_f64(k[(size_t)j * D + d]);
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
        double p = exp(s[j] - m) / l;
        if (probs)
            probs[j] = p;
        for (int d = 0; d < D; ++d)
            o[d] += p * bf16_to_f64(v[(size_t)j * D + d]);
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
            attend_row(qi, kb, vb, L, D, scale, s, o + (size_t)t * D, lse + t, pr);
        }
        free(s);
    }
    return failed ? -1 : 0;
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
