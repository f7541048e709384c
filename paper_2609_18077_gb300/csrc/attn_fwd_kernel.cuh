// Softmax attention forward for sm_103a (GB300): TMA-fed, tcgen05 tensor cores,
// accumulators and probabilities in tensor memory, warp-specialised.
//
// What it computes (vidax paper, Sec. 2 "3D RoPE, 3D VAEs, and flash
// attention"): out = softmax(scale * Q K^T) V and the natural-log row
// log-sum-exp, without ever storing the Sq x Skv score matrix, over
// [B, H, S, D] bf16 video tokens.  The varlen instance skips key tiles past a
// sample's valid text length and masks the ragged last tile (appendix Table 4:
// segment-id masking of padded text keys instead of a dense mask).  The
// segment instance (joint text-video attention, same appendix entry) lets
// query i attend key j iff their segment ids match: each unit visits only the
// key tiles of its list (segment_tiles.cuh) and compares ids element by
// element only on the tiles the list marks.  The window instance (windowed 3D
// attention, appendix Table 4's VAE decoder) takes its query tiles as 3-D
// bricks of the token grid and walks a regular grid of 3-D key boxes over the
// union of the unit's windows (window_tiles.cuh), through 5-D tensor maps,
// masking keys outside each row's window.
//
// Work unit: one (b*h, pair of 128-row query tiles).  The grid is persistent:
// one CTA per SM walks the units u = blockIdx.x, blockIdx.x + gridDim.x, ...
// The K/V stream runs on across units (a unit's last stage carries the next
// unit's K_0), each Q tile is reloaded as soon as the unit's last QK^T has
// run, and each O accumulator is handed to the next unit as soon as the
// epilogue holds it in registers, so one unit's start overlaps the previous
// unit's end.  Roles:
//   warps 0-3  softmax of query tile 0: thread = one query row (TMEM lane)
//   warps 4-7  softmax of query tile 1
//   warp  8    TMA producer: Q tiles once, then K_0 and the stages
//              (V_0, K_1), (V_1, K_2), ... through a ring of NSTAGE
//              two-tile stages (one full and one empty barrier per stage);
//              the next unit's Q tiles are prefetched into L2 meanwhile
//              (on units of at least Q_PREFETCH_MIN_TILES key tiles)
//   warp  9    tcgen05 issuer (one lane) and TMEM owner
// Tensor memory (512 columns x 128 lanes, fp32):
//   S_t = cols [128t, 128t+128): logits Q_t K_j^T; the probabilities P_t are
//         written back over its first 64 columns as packed bf16 pairs and fed
//         to the second GEMM straight from TMEM.
//   O_t = cols [256+128t, 256+128t+D): the running output accumulator.
// MMA order per key tile j (ping-pong between the two query tiles so that the
// softmax of one tile overlaps the GEMMs of the other):
//   ... PV_0(j)  S_0(j+1)  PV_1(j)  S_1(j+1) ...
// The issuing thread stalls on every barrier check (the tensor core holds
// about one MMA ahead of execution), so it checks only P_t per step: the
// softmax warps confirm that the step's V and next K have landed before they
// publish P.
// Online softmax in base 2 with a lazy maximum: a row's reference maximum m
// only moves when the tile maximum exceeds it by more than TAU (log2 units),
// so p <= 2^TAU and the O rescale in TMEM is rare after the first tiles.
//
// Normalisation.  The P V GEMM multiplies V by bf16-rounded weights r_j while
// the softmax sums the fp32 weights p_j.  In a row dominated by one key the
// mismatch r/p - 1 (up to 2^-8) would pass straight into O, so the divisor of
// O is the exact sum plus, for every key tile, the rounding residual r - p of
// that tile's largest weight in the row.  That makes the dominant weight
// exact at the cost of a few instructions per tile; the log-sum-exp uses the
// exact sum alone.
//
// Epilogue: O / l packed to bf16 by the softmax threads, one row each, and
// stored per thread; the text cross-attention instance, whose units are a few
// key tiles long, stores it through per-warp TMA stores from swizzled staging
// boxes instead (stages_out below).
//
// Every wait is bounded (globaltimer); on expiry the CTA records
// VDX_ERR_TIMEOUT in the device error word and skips the rest of its work.
// Before it exits, the producer waits for every TMA load it issued to land
// and the issuer for every tensor-core operation it issued to retire (both
// complete by themselves, so these waits cannot be stranded by another
// warp); only then is tensor memory freed and the CTA's shared memory, which
// those loads write and whose barriers they signal, given up.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <climits>
#include <cstdint>

#include "segment_tiles.cuh"
#include "sm103_ptx.cuh"
#include "window_tiles.cuh"

namespace vdx {

// Problem kinds (template parameter MODE of the kernel).
constexpr int MODE_DENSE = 0;    // all Skv keys
constexpr int MODE_VARLEN = 1;   // the first kv_lens[b] keys of sample b
constexpr int MODE_SEG = 2;      // the keys whose segment id equals the query's
constexpr int MODE_WIN = 3;      // the keys inside the query's 3D window (S = F*Hp*Wp grid tokens)
// Modes that visit key tiles from a list and may mask a row's every key so far.
__host__ __device__ constexpr bool listed(int mode) { return mode == MODE_SEG || mode == MODE_WIN; }

// Device error word, one per device, shared by every launch; taken (read and
// zeroed in one atomic exchange) by vdx_check_device_error.
//   bit 0: a bounded wait expired and the CTA gave up its work;
//   bit 1: the issuer's final wait for its tensor-core operations expired, so
//          tensor memory was released with operations possibly in flight;
//   bit 2: a TMA load issued by the producer had not landed when the CTA was
//          about to exit (its wait for the load expired).
// Bits 1 and 2 mean the GPU broke a completion guarantee; bit 0 alone means
// the work stopped cleanly.
__device__ unsigned int g_error_word;
constexpr unsigned ERR_WAIT_EXPIRED = 1u;
constexpr unsigned ERR_MMA_DRAIN = 2u;
constexpr unsigned ERR_LOADS_IN_FLIGHT = 4u;

constexpr int BM = 128;          // query rows per tile (= TMEM lanes)
constexpr int BN = 128;          // keys per tile
constexpr int NUM_THREADS = 320; // 8 softmax warps + producer + MMA
constexpr int PRODUCER_WARP = 8;
constexpr int MMA_WARP = 9;
constexpr float TAU = 8.0f;      // lazy-rescale threshold, log2 units
constexpr uint32_t TMEM_COLS = 512;
constexpr int Q_PREFETCH_MIN_TILES = 16;   // key tiles an item needs before the next Q is prefetched to L2

struct AttnParams {
    __nv_bfloat16 *out;
    float *lse;
    const int *kv_lens;   // varlen only
    int H;
    int Sq;
    int Skv;              // Skv (dense) or Skv_max (varlen)
    int q_pairs;          // ceil(ceil(Sq / BM) / 2)
    int units;            // B * H * q_pairs work units, handed out round-robin to the CTAs
    int out_align32;      // out is 32-byte aligned: write O with 256-bit stores
    // Split tail (0 parts: off).  The first full_rounds * gridDim.x units are
    // whole items; each of the tail_units remaining ones is cut into
    // split_parts key ranges, one per CTA, merged through the workspace.
    int split_parts;
    int full_rounds;
    int tail_units;
    float *ws_o;          // [tail_units][split_parts][2][BM][D] unnormalised fp32 accumulators
    float *ws_stats;      // [tail_units][split_parts][2][BM] float4 (m, l_exact, l_resid, -)
    int *ws_count;        // [tail_units] parts finished (zeroed before the launch)
    float scale_log2;     // scale * log2(e); never 0: |value| >= 1e-30
    uint64_t wait_limit_ns;
};

// Segment ids (MODE_SEG): q_seg [B, Sq], kv_seg [B, Skv]; per (b, query-tile
// pair) the key-tile list tlist[(b * q_pairs + qp) * n_kt + r], r < tcount[.].
// A kernel parameter of its own: with these fields inside AttnParams the
// register allocation of the dense and varlen kernels changed and the dense
// kernel measured 2 % slower.
struct SegParams {
    const int *q_seg;
    const int *kv_seg;
    const uint32_t *tlist;
    const int *tcount;
    int n_kt;             // key tiles of the whole sequence, ceil(Skv / BN)
    WinGrid win;          // MODE_WIN: grid and window; lists per query-tile pair, shared by (b, h)
};

// Shared-memory plan.  QBUF Q-tile pairs (2 = the next item's Q tiles load
// while the current item runs) and NSTAGE K/V stages of (V_j, next K).
template <int D, int QBUF, int NSTAGE_, bool OSTAGE = false>
struct Layout {
    static_assert(D == 64 || D == 128, "head dim");
    static constexpr int TILE_BYTES = BM * D * 2;           // one Q, K or V tile
    static constexpr int HALF_BYTES = BM * 128;              // one 64-column swizzle block
    static constexpr int NSTAGE = NSTAGE_;                   // K/V ring: stage = (V_j, next K)
    static constexpr int Q_OFF = 0;                          // Q buffer b, tile t at (2b + t) tiles
    static constexpr int KV_OFF = 2 * QBUF * TILE_BYTES;     // stage s: V at 2s, K at 2s+1 (tiles)
    static constexpr int BAR_OFF = KV_OFF + 2 * NSTAGE * TILE_BYTES;
    // barrier indices
    static constexpr int B_Q = 0;                            // [2 QBUF] Q tile (buffer b, tile t) landed
    static constexpr int B_QE = 2 * QBUF;                    // [2 QBUF] that Q tile free (its last QK^T ran)
    static constexpr int B_FULL = 4 * QBUF;                  // [NSTAGE] stage landed
    static constexpr int B_EMPTY = B_FULL + NSTAGE;          // [NSTAGE] stage consumed
    static constexpr int B_S = B_EMPTY + NSTAGE;             // [2] S_t ready
    static constexpr int B_P = B_S + 2;                      // [2] P_t written, O_t rescaled
    static constexpr int B_O = B_P + 2;                      // [2] last PV_t of a unit done
    static constexpr int B_OE = B_O + 2;                     // [2] O_t read out by the epilogue
    static constexpr int B_FIX = B_OE + 2;                   // varlen V tile staging
    static constexpr int B_DRAIN = B_FIX + 1;                // all MMAs retired
    static constexpr int B_MERGE = B_DRAIN + 1;              // [2] tail part written (8 warps) / merge decided
    static constexpr int NBARS = B_MERGE + 2;
    static constexpr int TMEM_PTR_OFF = BAR_OFF + NBARS * 8;
    static constexpr int ABORT_OFF = TMEM_PTR_OFF + 4;
    static constexpr int MERGE_OFF = ABORT_OFF + 4;          // "this CTA merges" flag
    // [NSTAGE][4] listed modes: list entry of each stage's V tile; MODE_WIN also
    // the grid position of its first key (t | h << 16, w)
    static constexpr int ENTRY_OFF = (MERGE_OFF + 4 + 15) / 16 * 16;
    // OSTAGE: per softmax warp, a 32-row x 128-byte (64-column) box of O in the
    // 128-byte swizzle of the output tensor map, written by the warp and stored
    // by TMA.
    static constexpr int OUT_BOX = 32 * 128;
    static constexpr int OUT_OFF = (ENTRY_OFF + 16 * NSTAGE + 1023) / 1024 * 1024;
    // Without OSTAGE 197.8 KB in all configurations: under the 196 KB
    // shared-memory carve-out (199,680 usable bytes), which leaves 60 KB of L1
    // for the spill slots.  With it 226 KB (the 228 KB carve-out).
    static constexpr int BYTES = OSTAGE ? OUT_OFF + 8 * OUT_BOX : ENTRY_OFF + 16 * NSTAGE;
    static constexpr int ALLOC = BYTES + 1024;               // slack for 1024-B alignment
};

// O leaves through TMA stores from shared memory in the text cross-attention
// instance, whose units are a few key tiles long: per-thread row stores (32
// rows of one warp hit 32 cache lines per instruction) then keep the load-store
// path busy long enough to delay the next unit's QK^T.  Elsewhere a unit runs
// hundreds of key steps and the per-thread stores cost nothing measurable.
template <int MODE>
__host__ __device__ constexpr bool stages_out()
{
    return MODE == MODE_VARLEN;
}

__device__ __forceinline__ bool wait_bounded(uint32_t bar, uint32_t parity, volatile int *abort_flag,
                                             uint64_t limit_ns)
{
    if (ptx::mbar_try_wait(bar, parity))
        return true;
    const uint64_t t0 = ptx::globaltimer_ns();
    for (uint32_t n = 1;; ++n) {
        if (ptx::mbar_try_wait(bar, parity))
            return true;
        if ((n & 255u) == 0) {
            if (*abort_flag)
                return false;
            if (ptx::globaltimer_ns() - t0 > limit_ns) {
                *abort_flag = 1;
                atomicOr(&g_error_word, ERR_WAIT_EXPIRED);
                return false;
            }
        }
    }
}

// Wait for a phase that completes by itself -- TMA bytes landing on a barrier
// whose arrivals were all made, or tensor-core operations retiring -- whatever
// the abort flag says.  Bounded all the same; false if the limit expired.
__device__ __forceinline__ bool wait_landed(uint32_t bar, uint32_t parity, uint64_t limit_ns)
{
    if (ptx::mbar_try_wait(bar, parity))
        return true;
    const uint64_t t0 = ptx::globaltimer_ns();
    while (!ptx::mbar_try_wait(bar, parity))
        if (ptx::globaltimer_ns() - t0 > limit_ns)
            return false;
    return true;
}

__device__ __forceinline__ float ex2(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi)
{
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t *>(&v);
}

__device__ __forceinline__ float round_bf16(float x)
{
    return __bfloat162float(__float2bfloat16_rn(x));
}

__device__ __forceinline__ float max3(float a, float b, float c)
{
    float d;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}

__device__ __forceinline__ float min3(float a, float b, float c)
{
    float d;
    asm("min.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}

// (d0, d1) = (a0, a1) * b + c on the paired fp32 datapath.
__device__ __forceinline__ void ffma2(float &d0, float &d1, float a0, float a1, float b, float c)
{
    asm("{\n\t.reg .b64 ra, rb, rc;\n\t"
        "mov.b64 ra, {%2, %3};\n\t"
        "mov.b64 rb, {%4, %4};\n\t"
        "mov.b64 rc, {%5, %5};\n\t"
        "fma.rn.f32x2 ra, ra, rb, rc;\n\t"
        "mov.b64 {%0, %1}, ra;\n\t}"
        : "=f"(d0), "=f"(d1)
        : "f"(a0), "f"(a1), "f"(b), "f"(c));
}

// (a0, a1) += (b0, b1) on the paired fp32 datapath.
__device__ __forceinline__ void fadd2(float &a0, float &a1, float b0, float b1)
{
    asm("{\n\t.reg .b64 ra, rb;\n\t"
        "mov.b64 ra, {%0, %1};\n\t"
        "mov.b64 rb, {%2, %3};\n\t"
        "add.rn.f32x2 ra, ra, rb;\n\t"
        "mov.b64 {%0, %1}, ra;\n\t}"
        : "+f"(a0), "+f"(a1)
        : "f"(b0), "f"(b1));
}

// S_t = Q_t K^T: M = 128 query rows, N = 128 keys, K = D in steps of 16.
// Both operands K-major, 128-byte swizzle, stored as D/64 blocks of
// 128 rows x 128 bytes; 8-row groups are 1024 bytes apart.  q_desc / k_desc
// describe the tile bases; a k-step adds its byte offset / 16 to the start
// address field (no carry: shared addresses stay below 256 KB).
template <int D>
__device__ __forceinline__ void issue_qk(uint32_t s_tmem, uint64_t q_desc, uint64_t k_desc)
{
    constexpr uint32_t idesc = ptx::idesc_bf16_f32(BM, BN, 0);
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
        const uint32_t off = ((kk >> 2) * (BM * 128) + (kk & 3) * 32) >> 4;
        ptx::mma_ss(s_tmem, q_desc + off, k_desc + off, idesc, kk > 0);
    }
}

// O_t (+)= P_t V: M = 128, N = D, K = 128 keys in steps of 16.  P comes from
// TMEM (16 bf16 = 8 columns per step); V is N-major ("MN-major"): each key row
// holds 64 contiguous head-dim values per 128-byte swizzled row, the two
// 64-column blocks are HALF_BYTES apart (LBO), 8-key groups 1024 bytes (SBO);
// a step of 16 keys advances 2048 bytes.
template <int D>
__device__ __forceinline__ void issue_pv(uint32_t o_tmem, uint32_t p_tmem, uint64_t v_desc, bool accumulate)
{
    constexpr uint32_t idesc = ptx::idesc_bf16_f32(BM, D, 1);
#pragma unroll
    for (int kk = 0; kk < BN / 16; ++kk)
        ptx::mma_ts(o_tmem, p_tmem + kk * 8, v_desc + kk * (2048 >> 4), idesc, (accumulate || kk > 0) ? 1u : 0u);
}

// Maximum (minimum for a negative scale) of the row's 128 raw logits.
__device__ __forceinline__ float row_extreme(const uint32_t (&s)[4][32], bool neg_scale)
{
    const float pad = neg_scale ? INFINITY : -INFINITY;
    float e0 = pad, e1 = pad, e2 = pad, e3 = pad;
#pragma unroll
    for (int c = 0; c < BN; c += 8) {
        float x[8];
#pragma unroll
        for (int i = 0; i < 8; ++i)
            x[i] = __uint_as_float(s[(c + i) >> 5][(c + i) & 31]);
        if (neg_scale) {
            e0 = min3(e0, x[0], x[1]); e1 = min3(e1, x[2], x[3]);
            e2 = min3(e2, x[4], x[5]); e3 = min3(e3, x[6], x[7]);
        } else {
            e0 = max3(e0, x[0], x[1]); e1 = max3(e1, x[2], x[3]);
            e2 = max3(e2, x[4], x[5]); e3 = max3(e3, x[6], x[7]);
        }
    }
    return neg_scale ? min3(fminf(e0, e1), e2, e3) : max3(fmaxf(e0, e1), e2, e3);
}

// p = 2^(x * scale_log2 - m) for the row's 128 logits, packed to bf16 pairs
// (even key in the low half, 64 TMEM columns); returns the fp32 sum of p.
__device__ __forceinline__ float row_probs(const uint32_t (&s)[4][32], uint32_t (&pk)[2][32], float sl2, float neg_m)
{
    float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
#pragma unroll
    for (int c = 0; c < BN; c += 4) {
        float x0, x1, x2, x3;
        ffma2(x0, x1, __uint_as_float(s[c >> 5][(c & 31) + 0]), __uint_as_float(s[c >> 5][(c & 31) + 1]), sl2,
              neg_m);
        ffma2(x2, x3, __uint_as_float(s[c >> 5][(c & 31) + 2]), __uint_as_float(s[c >> 5][(c & 31) + 3]), sl2,
              neg_m);
        const float p0 = ex2(x0), p1 = ex2(x1), p2 = ex2(x2), p3 = ex2(x3);
        fadd2(a0, a1, p0, p1);
        fadd2(a2, a3, p2, p3);
        pk[c >> 6][(c & 63) >> 1] = pack_bf16x2(p0, p1);
        pk[c >> 6][((c & 63) >> 1) + 1] = pack_bf16x2(p2, p3);
    }
    return (a0 + a1) + (a2 + a3);
}

// Merge of a split tail unit, run by the CTA that finishes its last part.
// Every part wrote, per query row, its unnormalised fp32 accumulator O_k and
// (m_k, le_k, lr_k): running maximum (log2 units), exact weight sum and
// rounding-residual sum.  With M = max m_k and w_k = 2^(m_k - M):
//   O = sum_k w_k O_k / sum_k w_k (le_k + lr_k),  LSE = (M + log2 sum_k w_k le_k) ln 2.
template <int D>
__device__ __noinline__ void merge_tail_parts(const AttnParams &p, int tail, int t, int row, int q_row, int bh,
                                              bool store, __nv_bfloat16 *orow, volatile int *last_flag,
                                              uint32_t bar_written, uint32_t bar_decided, volatile int *abort_flag)
{
    // All eight softmax warps wrote their rows of the part; publish them.  The
    // two waits are bounded, so a CTA that aborted elsewhere cannot hang here.
    const int lane = threadIdx.x & 31;
    __threadfence();
    __syncwarp();
    if (lane == 0)
        ptx::mbar_arrive(bar_written);
    if (threadIdx.x == 0) {
        int last = 0;
        if (wait_bounded(bar_written, 0, abort_flag, p.wait_limit_ns)) {
            const int done = atomicAdd(p.ws_count + tail, 1);
            last = done == p.split_parts - 1;
        }
        *last_flag = last;
        ptx::mbar_arrive(bar_decided);
    }
    if (!__all_sync(0xffffffffu, wait_bounded(bar_decided, 0, abort_flag, p.wait_limit_ns)) || !*last_flag)
        return;
    __threadfence();
    const int P = p.split_parts;
    auto slot = [&](int k) { return (tail * P + k) * 2 + t; };
    float M = -INFINITY;
    for (int k = 0; k < P; ++k)
        M = fmaxf(M, __ldcg(reinterpret_cast<const float4 *>(p.ws_stats) + slot(k) * BM + row).x);
    float le = 0.f, lc = 0.f;
    for (int k = 0; k < P; ++k) {
        const float4 st = __ldcg(reinterpret_cast<const float4 *>(p.ws_stats) + slot(k) * BM + row);
        const float wk = ex2(st.x - M);
        le += wk * st.y;
        lc += wk * (st.y + st.z);
    }
    const float inv = 1.f / lc;
#pragma unroll
    for (int c = 0; c < D / 32; ++c) {
        float acc[32];
#pragma unroll
        for (int i = 0; i < 32; ++i)
            acc[i] = 0.f;
        for (int k = 0; k < P; ++k) {
            const float wk = ex2(__ldcg(reinterpret_cast<const float4 *>(p.ws_stats) + slot(k) * BM + row).x - M);
            const float4 *src = reinterpret_cast<const float4 *>(p.ws_o + (static_cast<size_t>(slot(k)) * BM + row) * D +
                                                                 32 * c);
#pragma unroll
            for (int v = 0; v < 8; ++v) {
                const float4 x = __ldcg(src + v);
                acc[4 * v + 0] = fmaf(wk, x.x, acc[4 * v + 0]);
                acc[4 * v + 1] = fmaf(wk, x.y, acc[4 * v + 1]);
                acc[4 * v + 2] = fmaf(wk, x.z, acc[4 * v + 2]);
                acc[4 * v + 3] = fmaf(wk, x.w, acc[4 * v + 3]);
            }
        }
        if (store) {
            uint4 *dst = reinterpret_cast<uint4 *>(orow + 32 * c);
#pragma unroll
            for (int v = 0; v < 4; ++v)
                dst[v] = make_uint4(pack_bf16x2(acc[8 * v] * inv, acc[8 * v + 1] * inv),
                                    pack_bf16x2(acc[8 * v + 2] * inv, acc[8 * v + 3] * inv),
                                    pack_bf16x2(acc[8 * v + 4] * inv, acc[8 * v + 5] * inv),
                                    pack_bf16x2(acc[8 * v + 6] * inv, acc[8 * v + 7] * inv));
        }
    }
    if (store && p.lse)
        p.lse[static_cast<size_t>(bh) * p.Sq + q_row] = (M + __log2f(le)) * 0.69314718055994530942f;
}

// One work item of a CTA: a whole unit (b*h, query-tile pair) with key tiles
// [j0, j1) = [0, n_kv), or -- for the units of a short last round, when the
// host splits them -- one part of such a unit's key tiles (part >= 0).  In
// MODE_SEG, j indexes the unit's key-tile list rather than the key tiles.
struct Item {
    int bh;
    int qp;
    int kv_valid;
    int n_kv;      // key tiles of the whole unit (MODE_SEG: list entries)
    int j0, j1;    // key tiles of this item
    int part;      // -1: whole unit; else the part index within tail unit `tail`
    int tail;
    int list_off;  // MODE_SEG: offset of the unit's list in tlist
    bool ok;       // false past the CTA's last item
};

template <int MODE>
__device__ __forceinline__ Item unit_item(const AttnParams &p, const SegParams &sp, int u)
{
    Item w;
    w.bh = u / p.q_pairs;
    w.qp = u - w.bh * p.q_pairs;
    w.kv_valid = p.Skv;
    w.list_off = 0;
    if (MODE == MODE_VARLEN) {
        const int len = __ldg(p.kv_lens + w.bh / p.H);
        w.kv_valid = len < 0 ? 0 : (len > p.Skv ? p.Skv : len);
    }
    w.n_kv = (w.kv_valid + BN - 1) / BN;
    if (MODE == MODE_SEG) {
        const int pair = (w.bh / p.H) * p.q_pairs + w.qp;
        w.n_kv = __ldg(sp.tcount + pair);
        w.list_off = pair * sp.n_kt;
    }
    if (MODE == MODE_WIN) {
        const WinUnit u = win_unit(sp.win, w.qp);   // key boxes over the unit's window union
        w.n_kv = u.nbt * u.nbh * u.nbw;
    }
    w.j0 = 0;
    w.j1 = w.n_kv;
    w.part = -1;
    w.tail = 0;
    w.ok = true;
    return w;
}

// The i-th item of CTA `cta`: units cta, cta + G, ... and, in split mode,
// after full_rounds of them one part of a tail unit.
template <int MODE>
__device__ __forceinline__ Item item_at(const AttnParams &p, const SegParams &sp, int cta, int i)
{
    const int G = gridDim.x;
    Item w;
    w.ok = false;
    if (p.split_parts == 0) {
        const int u = cta + i * G;
        if (u < p.units)
            w = unit_item<MODE>(p, sp, u);
        return w;
    }
    if (i < p.full_rounds)
        return unit_item<MODE>(p, sp, cta + i * G);
    if (i == p.full_rounds && cta < p.tail_units * p.split_parts) {
        const int tail = cta / p.split_parts;
        const int part = cta - tail * p.split_parts;
        w = unit_item<MODE>(p, sp, p.full_rounds * G + tail);
        w.j0 = part * w.n_kv / p.split_parts;
        w.j1 = (part + 1) * w.n_kv / p.split_parts;
        w.part = part;
        w.tail = tail;
    }
    return w;
}

// List entry of position r of item w: in MODE_SEG the key tile and its mask
// bits (segment_tiles.cuh); otherwise r itself (the key tile, or in MODE_WIN
// the key box).
template <int MODE>
__device__ __forceinline__ uint32_t tile_entry(const SegParams &sp, const Item &w, int r)
{
    if (MODE == MODE_SEG)
        return __ldg(sp.tlist + w.list_off + r);
    return static_cast<uint32_t>(r);
}

// Where a K or V tile (or, in MODE_WIN, a key box) sits in its tensor map:
// (row, b*h) of the 3-D map, or (w, h, t, b*h) of the 5-D one.
struct TileAt {
    int bh;
    int c0, c1, c2;
};

template <int MODE>
__device__ __forceinline__ TileAt tile_at(const SegParams &sp, const Item &w, int j)
{
    TileAt a;
    a.bh = w.bh;
    if (MODE == MODE_WIN) {
        const WinUnit u = win_unit(sp.win, w.qp);
        win_box(sp.win, u, j, a.c2, a.c1, a.c0);
    } else {
        a.c0 = j * BN;
        a.c1 = a.c2 = 0;
    }
    return a;
}

// One 64-column half (x = 0 or 64) of a tile, through the map's dimensionality.
template <int MODE>
__device__ __forceinline__ void tma_tile(uint32_t dst, const CUtensorMap *map, uint32_t bar, int x, const TileAt &a)
{
    if (MODE == MODE_WIN)
        ptx::tma_load_5d(dst, map, bar, x, a.c0, a.c1, a.c2, a.bh);
    else
        ptx::tma_load_3d(dst, map, bar, x, a.c0, a.bh);
}

// Query tile t of item w: its 3-D tile (row) or, in MODE_WIN, its brick.
template <int MODE>
__device__ __forceinline__ TileAt q_tile_at(const SegParams &sp, const Item &w, int t)
{
    TileAt a;
    a.bh = w.bh;
    if (MODE == MODE_WIN) {
        const WinUnit u = win_unit(sp.win, w.qp);
        a.c0 = u.w0;
        a.c1 = u.h0;
        a.c2 = u.t0 + (t << sp.win.qlt);
    } else {
        a.c0 = (w.qp * 2 + t) * BM;
        a.c1 = a.c2 = 0;
    }
    return a;
}

template <int D, int MODE, int QBUF, int NSTAGE>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    attn_fwd_kernel(const __grid_constant__ CUtensorMap tmap_q, const __grid_constant__ CUtensorMap tmap_k,
                    const __grid_constant__ CUtensorMap tmap_v, const __grid_constant__ CUtensorMap tmap_o,
                    const AttnParams p, const __grid_constant__ SegParams sp)
{
    constexpr bool OSTAGE = stages_out<MODE>();
    using L = Layout<D, QBUF, NSTAGE, OSTAGE>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const uint32_t sbase = ptx::smem_u32(sm);
    auto bar = [&](int i) -> uint32_t { return sbase + L::BAR_OFF + 8 * i; };
    volatile int *abort_flag = reinterpret_cast<volatile int *>(sm + L::ABORT_OFF);
    const uint64_t limit = p.wait_limit_ns;
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int cta = blockIdx.x;

    if (threadIdx.x == 0) {
        for (int b = 0; b < 2 * QBUF; ++b) {
            ptx::mbar_init(bar(L::B_Q + b), 1);
            ptx::mbar_init(bar(L::B_QE + b), 1);
        }
        for (int t = 0; t < 2; ++t) {
            ptx::mbar_init(bar(L::B_S + t), 1);
            ptx::mbar_init(bar(L::B_P + t), 4);    // one arrive per softmax warp
            ptx::mbar_init(bar(L::B_O + t), 1);
            ptx::mbar_init(bar(L::B_OE + t), 4);   // one arrive per softmax warp
        }
        for (int i = 0; i < L::NSTAGE; ++i) {
            ptx::mbar_init(bar(L::B_FULL + i), 1);
            ptx::mbar_init(bar(L::B_EMPTY + i), 1);
        }
        ptx::mbar_init(bar(L::B_FIX), 1);
        ptx::mbar_init(bar(L::B_DRAIN), 1);
        ptx::mbar_init(bar(L::B_MERGE + 0), 8);
        ptx::mbar_init(bar(L::B_MERGE + 1), 1);
        *abort_flag = 0;
        ptx::fence_barrier_init();
        ptx::fence_proxy_async_smem();
    }
    if (warp == MMA_WARP) {
        ptx::tmem_alloc(sbase + L::TMEM_PTR_OFF, TMEM_COLS);
        ptx::tmem_relinquish();
    }
    if (warp == PRODUCER_WARP && lane == 0) {
        ptx::tma_prefetch_desc(&tmap_q);
        ptx::tma_prefetch_desc(&tmap_k);
        ptx::tma_prefetch_desc(&tmap_v);
        if (OSTAGE)
            ptx::tma_prefetch_desc(&tmap_o);
    }
    ptx::tc_fence_before_sync();
    __syncthreads();
    ptx::tc_fence_after_sync();
    const uint32_t tmem = *reinterpret_cast<volatile uint32_t *>(sm + L::TMEM_PTR_OFF);

    if (warp == PRODUCER_WARP) {
        // ------------------------------------------------------------ TMA producer
        // Stage g of this CTA's stream holds (V_j, next K): the j-th value tile
        // of an item and the key tile its GEMMs need next -- K_{j+1} of the
        // same item or the first key tile of the next item with keys.  Stage 0
        // holds that first key tile alone.
        const uint64_t q_policy = ptx::policy_evict_first();
        auto next_with_keys = [&](int i) {
            for (++i;; ++i) {
                const Item w = item_at<MODE>(p, sp, cta, i);
                if (!w.ok)
                    return -1;
                if (w.j1 > w.j0)
                    return i;
            }
        };
        int g = 0;          // stages armed so far
        int fixes = 0;      // B_FIX phases completed
        bool fix_pending = false;   // a B_FIX phase armed but not seen complete
        uint32_t q_armed = 0;       // bit b: Q barrier b armed at least once
        uint32_t q_parity = 0;      // bit b: parity of Q barrier b's last armed phase
        bool ok = true;
        // load stage g: V tile va if has_v, K tile ka if has_k.
        // Listed modes: the V tile's list entry (MODE_WIN: the key box's
        // origin) goes to the stage's slot before the full barrier is armed
        // (its arrive releases the slot to the softmax, which reads it after
        // its wait on that barrier; the slot is rewritten only after the stage
        // is released, i.e. after that read).
        auto stage = [&](const TileAt &va, bool has_v, int v_valid, const TileAt &ka, bool has_k,
                         uint32_t ventry) -> bool {
            const int st = g % L::NSTAGE;
            const int rnd = g / L::NSTAGE;
            if (rnd > 0 &&
                !__all_sync(0xffffffffu, wait_bounded(bar(L::B_EMPTY + st), (rnd - 1) & 1, abort_flag, limit)))
                return false;
            ++g;
            const uint32_t vdst = sbase + L::KV_OFF + (2 * st) * L::TILE_BYTES;
            const uint32_t kdst = vdst + L::TILE_BYTES;
            const bool fix = MODE == MODE_VARLEN && has_v && v_valid < BN;
            if (fix) {
                // A padded sample's last V tile: rows past the valid length may
                // hold any bits (NaN included) and 0 * NaN = NaN inside the
                // GEMM, so stage the tile, zero those rows, then publish.
                // The stage's K tile loads meanwhile: its bytes count on the
                // full barrier, whose one arrival comes after the zeroing.
                if (lane == 0) {
                    ptx::mbar_arrive_expect_tx(bar(L::B_FIX), L::TILE_BYTES);
                    for (int h = 0; h < D / 64; ++h)
                        tma_tile<MODE>(vdst + h * L::HALF_BYTES, &tmap_v, bar(L::B_FIX), h * 64, va);
                    if (has_k) {
                        ptx::mbar_expect_tx(bar(L::B_FULL + st), L::TILE_BYTES);
                        for (int h = 0; h < D / 64; ++h)
                            tma_tile<MODE>(kdst + h * L::HALF_BYTES, &tmap_k, bar(L::B_FULL + st), h * 64, ka);
                    }
                }
                fix_pending = true;
                if (!__all_sync(0xffffffffu, wait_bounded(bar(L::B_FIX), fixes & 1, abort_flag, limit))) {
                    // Give the stage its one arrival, so that its phase completes
                    // once the K bytes land and the drain below can see them land.
                    if (lane == 0)
                        ptx::mbar_arrive(bar(L::B_FULL + st));
                    return false;
                }
                fix_pending = false;
                ++fixes;
                // Lane l zeroes 16-byte chunk l % 8 of rows v_valid + l / 8,
                // + 4, + 8, ... of each 64-column block (a row is 8 chunks; no
                // division: this runs on the producer's critical path).
                uint8_t *slot_ptr = sm + L::KV_OFF + (2 * st) * L::TILE_BYTES + (lane & 7) * 16;
                for (int h = 0; h < D / 64; ++h)
                    for (int r = v_valid + (lane >> 3); r < BN; r += 4)
                        *reinterpret_cast<uint4 *>(slot_ptr + h * L::HALF_BYTES + r * 128) = make_uint4(0u, 0u, 0u, 0u);
                ptx::fence_proxy_async_smem();
                __syncwarp();
            }
            if (lane == 0) {
                const uint32_t bytes = fix ? 0u : (has_v + has_k) * L::TILE_BYTES;
                if (listed(MODE) && has_v) {
                    volatile uint32_t *slot = reinterpret_cast<volatile uint32_t *>(sm + L::ENTRY_OFF) + 4 * st;
                    slot[0] = ventry;
                    if (MODE == MODE_WIN) {
                        // the key box's origin (t | h << 16, w)
                        slot[1] = static_cast<uint32_t>(va.c2) | (static_cast<uint32_t>(va.c1) << 16);
                        slot[2] = static_cast<uint32_t>(va.c0);
                    }
                }
                if (bytes) {
                    ptx::mbar_arrive_expect_tx(bar(L::B_FULL + st), bytes);
                    for (int h = 0; h < D / 64; ++h) {
                        if (has_v && !fix)
                            tma_tile<MODE>(vdst + h * L::HALF_BYTES, &tmap_v, bar(L::B_FULL + st), h * 64, va);
                        if (has_k)
                            tma_tile<MODE>(kdst + h * L::HALF_BYTES, &tmap_k, bar(L::B_FULL + st), h * 64, ka);
                    }
                } else {
                    ptx::mbar_arrive(bar(L::B_FULL + st));
                }
            }
            return true;
        };
        int i = 0;
        {
            const Item w0 = item_at<MODE>(p, sp, cta, 0);
            if (!w0.ok)
                i = -1;
            else if (w0.j1 == w0.j0)
                i = next_with_keys(0);
        }
        if (i >= 0) {
            const Item w = item_at<MODE>(p, sp, cta, i);
            const TileAt none{0, 0, 0, 0};
            ok = stage(none, false, BN, tile_at<MODE>(sp, w, static_cast<int>(tile_entry<MODE>(sp, w, w.j0) &
                                                                              SEG_TILE_BITS)),
                       true, 0u);
        }
        for (int iq = 0; ok && i >= 0; ++iq) {
            const Item w = item_at<MODE>(p, sp, cta, i);
            const int ni = next_with_keys(i);
            const int qb = iq % QBUF;
            // Each Q tile of buffer qb is free once its previous item's last
            // QK^T ran; tile 0's load starts without waiting for tile 1's.
            for (int t = 0; ok && t < 2; ++t) {
                if (iq >= QBUF)
                    ok = __all_sync(0xffffffffu, wait_bounded(bar(L::B_QE + 2 * qb + t), ((iq / QBUF) - 1) & 1,
                                                              abort_flag, limit));
                if (ok && lane == 0) {
                    ptx::mbar_arrive_expect_tx(bar(L::B_Q + 2 * qb + t), L::TILE_BYTES);
                    const TileAt qa = q_tile_at<MODE>(sp, w, t);
                    const uint32_t qdst = sbase + L::Q_OFF + (2 * qb + t) * L::TILE_BYTES;
                    // A Q tile is read once: first in line for eviction from
                    // L2, so that it does not push out the keys and values
                    // other CTAs still stream (13 % fewer DRAM reads per call
                    // at S = 75600, same time).
                    for (int h = 0; h < D / 64; ++h) {
                        if (MODE == MODE_WIN)
                            tma_tile<MODE>(qdst + h * L::HALF_BYTES, &tmap_q, bar(L::B_Q + 2 * qb + t), h * 64, qa);
                        else
                            ptx::tma_load_3d_hint(qdst + h * L::HALF_BYTES, &tmap_q, bar(L::B_Q + 2 * qb + t), h * 64,
                                                  qa.c0, qa.bh, q_policy);
                    }
                }
                if (ok) {
                    const uint32_t bit = 1u << (2 * qb + t);
                    q_armed |= bit;
                    q_parity = (q_parity & ~bit) | (((iq / QBUF) & 1) ? bit : 0u);
                }
            }
            if (!ok)
                break;
            Item nw;
            nw.ok = false;
            if (ni >= 0)
                nw = item_at<MODE>(p, sp, cta, ni);
            // The next item's Q tiles can load only once this item's last QK^T
            // ran; start bringing them to L2 now so that load is short (a hint:
            // nothing waits for it).  Only items of many key tiles leave the
            // hint time to land: on items of a few tiles (text keys) it ran
            // 2.4 % slower than none, on items of hundreds 1.4 % faster.
            if (lane == 0 && nw.ok && w.j1 - w.j0 >= Q_PREFETCH_MIN_TILES)
                for (int t = 0; t < 2; ++t) {
                    const TileAt qa = q_tile_at<MODE>(sp, nw, t);
                    for (int h = 0; h < D / 64; ++h) {
                        if (MODE == MODE_WIN)
                            ptx::tma_prefetch_5d(&tmap_q, h * 64, qa.c0, qa.c1, qa.c2, qa.bh);
                        else
                            ptx::tma_prefetch_3d(&tmap_q, h * 64, qa.c0, qa.bh);
                    }
                }
            uint32_t ve = tile_entry<MODE>(sp, w, w.j0);
            for (int j = w.j0; ok && j < w.j1; ++j) {
                const bool last = j + 1 == w.j1;
                // MODE_SEG: the list entry is read before the stage's empty wait
                const uint32_t ke = last ? (nw.ok ? tile_entry<MODE>(sp, nw, nw.j0) : 0u) : tile_entry<MODE>(sp, w, j + 1);
                const bool has_k = !(last && !nw.ok);
                const int kj = static_cast<int>(ke & SEG_TILE_BITS);
                const int vj = static_cast<int>(ve & SEG_TILE_BITS);
                const TileAt ka = has_k ? tile_at<MODE>(sp, last ? nw : w, kj) : TileAt{0, 0, 0, 0};
                ok = stage(tile_at<MODE>(sp, w, vj), true, w.kv_valid - vj * BN, ka, has_k, ve);
                ve = ke;
            }
            i = ni;
        }
        // Every TMA load above completes on a barrier in this CTA's shared
        // memory, and none may still be in flight when the CTA exits: after an
        // abort the consumers stop waiting for them, so the producer waits for
        // the last armed phase of every barrier it loads to (all its arrivals
        // were made, so the phase completes by itself once the bytes land).
        // Without an abort every such phase was consumed and these checks pass
        // at once.
        if (lane == 0) {
            bool landed = true;
            for (int st = 0; st < L::NSTAGE; ++st)
                if (g > st)
                    landed &= wait_landed(bar(L::B_FULL + st), ((g - 1 - st) / L::NSTAGE) & 1, limit);
            for (int b = 0; b < 2 * QBUF; ++b)
                if ((q_armed >> b) & 1u)
                    landed &= wait_landed(bar(L::B_Q + b), (q_parity >> b) & 1u, limit);
            if (fix_pending)
                landed &= wait_landed(bar(L::B_FIX), fixes & 1, limit);
            if (!landed)
                atomicOr(&g_error_word, ERR_LOADS_IN_FLIGHT);
        }
        __syncwarp();
    } else if (warp == MMA_WARP) {
        // ------------------------------------------------------------ tcgen05 issuer
        if (lane == 0) {
            const uint64_t dq_base = ptx::smem_desc_sw128(sbase + L::Q_OFF, 16, 1024);
            constexpr uint32_t TILE16 = L::TILE_BYTES >> 4;
            const uint64_t dk = ptx::smem_desc_sw128(sbase + L::KV_OFF + L::TILE_BYTES, 16, 1024);
            const uint64_t dv = ptx::smem_desc_sw128(sbase + L::KV_OFF, L::HALF_BYTES, 1024);
            constexpr uint32_t STAGE16 = (2 * L::TILE_BYTES) >> 4;
            const uint32_t s0 = tmem, s1 = tmem + 128, o0 = tmem + 256, o1 = tmem + 384;
            int g = 1;         // stage holding the current item's (V_j0, next K)
            int pc = 0;        // P phases consumed (per tile, identical)
            int iq = 0;        // items with keys so far
            bool ok = true;
            for (int i = 0; ok; ++i) {
                const Item w = item_at<MODE>(p, sp, cta, i);
                if (!w.ok)
                    break;
                const int n = w.j1 - w.j0;
                if (n == 0)
                    continue;
                if (iq == 0)
                    ok = wait_bounded(bar(L::B_FULL + 0), 0, abort_flag, limit);   // first key tile
                const int qb = iq % QBUF;
                const int qph = (iq / QBUF) & 1;
                // Each tile's first QK^T as soon as that tile's Q landed.
                ok = ok && wait_bounded(bar(L::B_Q + 2 * qb), qph, abort_flag, limit);
                if (!ok)
                    break;
                const uint64_t dq0 = dq_base + (2 * qb) * TILE16;
                const uint64_t dq1 = dq_base + (2 * qb + 1) * TILE16;
                // The item's first key tile sits in the stage before its first.
                const int st_k0 = (g - 1) % L::NSTAGE;
                ptx::tc_fence_after_sync();
                issue_qk<D>(s0, dq0, dk + st_k0 * STAGE16);
                ptx::mma_commit(bar(L::B_S + 0));
                if (!(ok = wait_bounded(bar(L::B_Q + 2 * qb + 1), qph, abort_flag, limit)))
                    break;
                ptx::tc_fence_after_sync();
                issue_qk<D>(s1, dq1, dk + st_k0 * STAGE16);
                ptx::mma_commit(bar(L::B_S + 1));
                // That stage also carried the previous item's last V: both are done now.
                ptx::mma_commit(bar(L::B_EMPTY + st_k0));
                if (n == 1) {
                    ptx::mma_commit(bar(L::B_QE + 2 * qb));
                    ptx::mma_commit(bar(L::B_QE + 2 * qb + 1));
                }
                for (int r = 0; r < n; ++r, ++pc) {
                    const int st = (g + r) % L::NSTAGE;
                    const uint64_t vd = dv + st * STAGE16;
                    const uint64_t kd = dk + st * STAGE16;
                    const bool more = r + 1 < n;
                    if (!(ok = wait_bounded(bar(L::B_P + 0), pc & 1, abort_flag, limit)))
                        break;
                    if (r == 0 && iq > 0 && !(ok = wait_bounded(bar(L::B_OE + 0), (iq - 1) & 1, abort_flag, limit)))
                        break;
                    ptx::tc_fence_after_sync();
                    issue_pv<D>(o0, s0, vd, r > 0);
                    if (more) {
                        issue_qk<D>(s0, dq0, kd);
                        ptx::mma_commit(bar(L::B_S + 0));
                        if (r + 2 == n)
                            ptx::mma_commit(bar(L::B_QE + 2 * qb));
                    } else {
                        ptx::mma_commit(bar(L::B_O + 0));
                    }
                    if (!(ok = wait_bounded(bar(L::B_P + 1), pc & 1, abort_flag, limit)))
                        break;
                    if (r == 0 && iq > 0 && !(ok = wait_bounded(bar(L::B_OE + 1), (iq - 1) & 1, abort_flag, limit)))
                        break;
                    ptx::tc_fence_after_sync();
                    issue_pv<D>(o1, s1, vd, r > 0);
                    if (more) {
                        issue_qk<D>(s1, dq1, kd);
                        ptx::mma_commit(bar(L::B_S + 1));
                        if (r + 2 == n)
                            ptx::mma_commit(bar(L::B_QE + 2 * qb + 1));
                        ptx::mma_commit(bar(L::B_EMPTY + st));
                    } else {
                        ptx::mma_commit(bar(L::B_O + 1));
                    }
                }
                g += n;
                ++iq;
            }
            // Retire every MMA this thread issued (and with them the arrivals
            // their commits make on this CTA's barriers) before TMEM is
            // released.  They need nothing from other warps, so they retire
            // within microseconds.  Should this wait still expire, bit 1 of
            // the error word records it and tensor memory is released all the
            // same: a CTA that exits holding tensor memory would leave every
            // later allocation on its multiprocessor waiting forever.
            ptx::mma_commit(bar(L::B_DRAIN));
            if (!wait_landed(bar(L::B_DRAIN), 0, limit))
                atomicOr(&g_error_word, ERR_MMA_DRAIN);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------ softmax warps
        const int t = warp >> 2;                 // query tile of this group
        const int wq = warp & 3;                 // TMEM lane quarter of this warp
        const int row = wq * 32 + lane;          // query row within the tile
        const uint32_t lane_addr = tmem + (static_cast<uint32_t>(wq * 32) << 16);
        const uint32_t s_addr = lane_addr + 128 * t;
        const uint32_t o_addr = lane_addr + 256 + 128 * t;
        const float sl2 = p.scale_log2;
        const bool neg_scale = sl2 < 0.f;
        // MODE_WIN: the combs of window_mask and its cache of t-range words
        const uint32_t comb_w = MODE == MODE_WIN ? repeat32(1u, sp.win.klw) : 0u;
        const uint32_t comb_s = MODE == MODE_WIN ? repeat32(1u, sp.win.klh + sp.win.klw) : 0u;
        int win_tc = INT_MIN;
        uint32_t win_tm[4] = {0u, 0u, 0u, 0u};
        int g = 1;      // stage of the current item's (V_j0, next K)
        int sc = 0;     // S phases consumed
        int iq = 0;     // items with keys so far
        bool ok = true;

        for (int i = 0; ok; ++i) {
            const Item w = item_at<MODE>(p, sp, cta, i);
            win_tc = INT_MIN;   // the row's window changes with the unit
            if (!w.ok)
                break;
            // This row's query: its token index q_row (stores and LSE) and, in
            // MODE_WIN, its window (one packed axis per word) for the whole unit;
            // a brick row outside the grid stores nothing and sees no key.
            int q_row = (w.qp * 2 + t) * BM + row;
            bool store = q_row < p.Sq;
            uint32_t win_t = 0, win_h = 0, win_w = 0;
            if (MODE == MODE_WIN) {
                const WinUnit u = win_unit(sp.win, w.qp);
                const int pw = u.w0 + (row & ((1 << sp.win.qlw) - 1));
                const int ph = u.h0 + ((row >> sp.win.qlw) & ((1 << sp.win.qlh) - 1));
                const int pt = u.t0 + (t << sp.win.qlt) + (row >> (sp.win.qlw + sp.win.qlh));
                store = pt < sp.win.F && ph < sp.win.Hp && pw < sp.win.Wp;
                q_row = store ? (pt * sp.win.Hp + ph) * sp.win.Wp + pw : 0;
                packed_window(sp.win, pt, ph, pw, win_t, win_h, win_w);
            }
            __nv_bfloat16 *orow = p.out + (static_cast<size_t>(w.bh) * p.Sq + (store ? q_row : 0)) * D;
            if (w.j1 == w.j0) {
                if (store) {
#pragma unroll
                    for (int c = 0; c < D / 8; ++c)
                        reinterpret_cast<uint4 *>(orow)[c] = make_uint4(0u, 0u, 0u, 0u);
                    if (p.lse)
                        p.lse[static_cast<size_t>(w.bh) * p.Sq + q_row] = -INFINITY;
                }
                continue;
            }
            float m_used = -INFINITY;
            float l_exact = 0.f;   // sum of the fp32 weights: the log-sum-exp
            float l_resid = 0.f;   // sum over tiles of r - p for each tile's largest weight
            for (int j = w.j0; j < w.j1; ++j, ++sc) {
                if (!(ok = __all_sync(0xffffffffu, wait_bounded(bar(L::B_S + t), sc & 1, abort_flag, limit))))
                    break;
                ptx::tc_fence_after_sync();
                const int gj = g + (j - w.j0);
                // MODE_WIN: the list entry comes with the stage's full barrier, so
                // that wait comes first here; the row's 128-key window mask is
                // then built while the logits are not yet in registers.
                uint32_t wmask[4] = {0u, 0u, 0u, 0u};
                if (MODE == MODE_WIN) {
                    if (!(ok = __all_sync(0xffffffffu, wait_bounded(bar(L::B_FULL + gj % L::NSTAGE),
                                                                    (gj / L::NSTAGE) & 1, abort_flag, limit))))
                        break;
                    const volatile uint32_t *slot =
                        reinterpret_cast<volatile uint32_t *>(sm + L::ENTRY_OFF) + 4 * (gj % L::NSTAGE);
                    const uint32_t th = slot[1];
                    window_mask(sp.win, win_t, win_h, win_w, static_cast<int>(th & 0xFFFFu),
                                static_cast<int>(th >> 16), static_cast<int>(slot[2]), comb_w, comb_s, win_tc, win_tm,
                                wmask);
                }
                uint32_t s[4][32];
#pragma unroll
                for (int c = 0; c < 4; ++c)
                    ptx::tmem_ld32(s_addr + 32 * c, s[c]);
                // The stage (V_j, next K) must have landed before P_t(j) is
                // published; checked here, under the TMEM load latency.
                if (MODE != MODE_WIN &&
                    !(ok = __all_sync(0xffffffffu, wait_bounded(bar(L::B_FULL + gj % L::NSTAGE),
                                                                (gj / L::NSTAGE) & 1, abort_flag, limit)))) {
                    ptx::tmem_wait_ld();
                    break;
                }
                ptx::tmem_wait_ld();

                int kt = j;   // key tile
                bool seg_mask = false;
                if (MODE == MODE_SEG) {
                    // the stage's list entry, published with its full barrier
                    const uint32_t entry = reinterpret_cast<volatile uint32_t *>(sm + L::ENTRY_OFF)[4 * (gj % L::NSTAGE)];
                    kt = static_cast<int>(entry & SEG_TILE_BITS);
                    seg_mask = (entry >> (SEG_MASK_SHIFT + t)) & 1u;
                }
                const int valid = w.kv_valid - kt * BN;
                if (MODE != MODE_WIN && valid < BN) {
                    // Ragged last tile: keys past the end (or past the sample's
                    // text length, whatever their bits) become -inf logits
                    // after scaling, i.e. weight exactly 0.  scale_log2 is never
                    // 0 (the host raises it to 1e-30), so inf * scale stays inf.
                    const uint32_t pad = neg_scale ? 0x7F800000u : 0xFF800000u;
#pragma unroll
                    for (int c = 0; c < BN; ++c)
                        s[c >> 5][c & 31] = c < valid ? s[c >> 5][c & 31] : pad;
                }
                if (MODE == MODE_SEG && seg_mask) {
                    // Keys of another segment get the masked logit too.  Lane
                    // l reads the ids of keys 32e + l and the warp shares them by
                    // shuffles (a marked tile is rare: segment borders only, so
                    // the load latency is taken here rather than kept in flight).
                    const uint32_t pad = neg_scale ? 0x7F800000u : 0xFF800000u;
                    const size_t b = static_cast<size_t>(w.bh / p.H);
                    const int my_seg = store ? __ldg(sp.q_seg + b * p.Sq + q_row) : 0;
                    const int *kseg = sp.kv_seg + b * p.Skv;
                    int ids[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const int c = kt * BN + e * 32 + lane;
                        ids[e] = c < p.Skv ? __ldg(kseg + c) : 0;
                    }
#pragma unroll
                    for (int c = 0; c < BN; ++c) {
                        const int kid = __shfl_sync(0xffffffffu, ids[c >> 5], c & 31);
                        s[c >> 5][c & 31] = kid == my_seg ? s[c >> 5][c & 31] : pad;
                    }
                }
                if (MODE == MODE_WIN) {
                    // keys outside this row's window (or the grid) get the masked logit
                    const uint32_t pad = neg_scale ? 0x7F800000u : 0xFF800000u;
#pragma unroll
                    for (int c = 0; c < BN; ++c)
                        s[c >> 5][c & 31] = (wmask[c >> 5] >> (c & 31)) & 1u ? s[c >> 5][c & 31] : pad;
                }
                const float ext = row_extreme(s, neg_scale);
                const float m_tile = ext * sl2;
                const float m_new = fmaxf(m_used, m_tile);
                const bool need = m_new > m_used + TAU;
                float factor = 1.f;
                if (need) {
                    factor = ex2(m_used - m_new);
                    m_used = m_new;
                }
                // MODE_SEG: a row whose keys so far were all masked keeps
                // m_used = -inf; its weights are 2^-inf = 0, not 2^(-inf + inf).
                const float neg_m = (listed(MODE) && m_used == -INFINITY) ? 0.f : -m_used;
                // the tile's largest weight, computed exactly as in row_probs
                const float p_top = ex2(fmaf(ext, sl2, neg_m));
                l_exact *= factor;
                l_resid = l_resid * factor + (round_bf16(p_top) - p_top);
                uint32_t pk[2][32];
                l_exact += row_probs(s, pk, sl2, neg_m);
                ptx::tmem_st32(s_addr, pk[0]);
                ptx::tmem_st32(s_addr + 32, pk[1]);
                if (j > w.j0 && __any_sync(0xffffffffu, need)) {
                    // O_t is idle here: S_t(j) was committed after PV_t(j-1), and
                    // PV_t(j) waits for the arrive below.  Done after P so that the
                    // logits' registers are free.
#pragma unroll
                    for (int c = 0; c < D / 32; ++c) {
                        uint32_t r[32];
                        ptx::tmem_ld32(o_addr + 32 * c, r);
                        ptx::tmem_wait_ld();
#pragma unroll
                        for (int k2 = 0; k2 < 32; ++k2)
                            r[k2] = __float_as_uint(__uint_as_float(r[k2]) * factor);
                        ptx::tmem_st32(o_addr + 32 * c, r);
                    }
                }
                ptx::tmem_wait_st();
                ptx::tc_fence_before_sync();
                __syncwarp();
                if (lane == 0)
                    ptx::mbar_arrive(bar(L::B_P + t));
            }
            if (!ok)
                break;

            // -------------------------------------------------------- epilogue
            if (!(ok = __all_sync(0xffffffffu, wait_bounded(bar(L::B_O + t), iq & 1, abort_flag, limit))))
                break;
            ptx::tc_fence_after_sync();
            if (w.part >= 0) {
                // Part of a split tail unit: the unnormalised fp32 accumulator
                // and this row's statistics go to the workspace; the last part
                // to finish merges the parts of the unit.
                const int slot = (w.tail * p.split_parts + w.part) * 2 + t;
                float *orow_ws = p.ws_o + (static_cast<size_t>(slot) * BM + row) * D;
#pragma unroll
                for (int c = 0; c < D / 32; ++c) {
                    uint32_t r[32];
                    ptx::tmem_ld32(o_addr + 32 * c, r);
                    ptx::tmem_wait_ld();
#pragma unroll
                    for (int v = 0; v < 4; ++v)
                        ptx::st_global_v8(orow_ws + 32 * c + 8 * v, &r[8 * v]);
                }
                reinterpret_cast<float4 *>(p.ws_stats)[slot * BM + row] = make_float4(m_used, l_exact, l_resid, 0.f);
                ptx::tc_fence_before_sync();
                __syncwarp();
                if (lane == 0)
                    ptx::mbar_arrive(bar(L::B_OE + t));
                merge_tail_parts<D>(p, w.tail, t, row, q_row, w.bh, store, orow,
                                    reinterpret_cast<volatile int *>(sm + L::MERGE_OFF), bar(L::B_MERGE),
                                    bar(L::B_MERGE + 1), abort_flag);
            } else {
                // MODE_SEG: a row with no key of its segment has l = 0 and O = 0.
                const float inv_l = (listed(MODE) && !(l_exact > 0.f)) ? 0.f : 1.f / (l_exact + l_resid);
                uint32_t w16[D / 32][16];
#pragma unroll
                for (int c = 0; c < D / 32; ++c) {
                    uint32_t r[32];
                    ptx::tmem_ld32(o_addr + 32 * c, r);
                    ptx::tmem_wait_ld();
#pragma unroll
                    for (int k2 = 0; k2 < 16; ++k2)
                        w16[c][k2] = pack_bf16x2(__uint_as_float(r[2 * k2]) * inv_l,
                                                 __uint_as_float(r[2 * k2 + 1]) * inv_l);
                }
                // O_t is in registers: hand the accumulator to the next item's
                // GEMMs before the global stores.
                ptx::tc_fence_before_sync();
                __syncwarp();
                if (lane == 0)
                    ptx::mbar_arrive(bar(L::B_OE + t));
                if (OSTAGE) {
                    // This warp's 32 rows through its staging box, 64 columns at a
                    // time: chunk c (16 bytes) of row r sits at chunk c ^ (r & 7).
                    const uint32_t stg = sbase + L::OUT_OFF + (4 * t + wq) * L::OUT_BOX;
                    const int row0 = (w.qp * 2 + t) * BM + wq * 32;
#pragma unroll
                    for (int h = 0; h < D / 64; ++h) {
                        if (lane == 0)
                            ptx::bulk_wait_read_all();   // the previous box was read out
                        __syncwarp();
#pragma unroll
                        for (int c = 0; c < 8; ++c) {
                            const uint32_t *src = &w16[2 * h + (c >> 2)][4 * (c & 3)];
                            ptx::st_shared_v4(stg + lane * 128 + ((c ^ (lane & 7)) << 4), src[0], src[1], src[2],
                                              src[3]);
                        }
                        ptx::fence_proxy_async_smem();
                        __syncwarp();
                        if (lane == 0 && row0 < p.Sq) {   // rows past Sq are clipped by the store
                            ptx::tma_store_3d(&tmap_o, stg, h * 64, row0, w.bh);
                            ptx::bulk_commit_group();
                        }
                    }
                    if (store && p.lse)
                        p.lse[static_cast<size_t>(w.bh) * p.Sq + q_row] =
                            (m_used + __log2f(l_exact)) * 0.69314718055994530942f;
                } else if (store) {
                    if (p.out_align32) {
                        // 32-byte stores: each fills a whole sector of the row.
#pragma unroll
                        for (int c = 0; c < D / 32; ++c)
#pragma unroll
                            for (int v = 0; v < 2; ++v)
                                ptx::st_global_v8(orow + 32 * c + 16 * v, &w16[c][8 * v]);
                    } else {
#pragma unroll
                        for (int c = 0; c < D / 32; ++c) {
                            uint4 *dst = reinterpret_cast<uint4 *>(orow + 32 * c);
#pragma unroll
                            for (int v = 0; v < 4; ++v)
                                dst[v] = make_uint4(w16[c][4 * v], w16[c][4 * v + 1], w16[c][4 * v + 2],
                                                    w16[c][4 * v + 3]);
                        }
                    }
                    if (p.lse)
                        p.lse[static_cast<size_t>(w.bh) * p.Sq + q_row] =
                            (m_used + __log2f(l_exact)) * 0.69314718055994530942f;
                }
            }
            g += w.j1 - w.j0;
            ++iq;
        }
        // An abort can leave this warp's tensor-memory loads or stores in
        // flight; none may remain when the memory is released below.  Nor may
        // an output store still be reading its staging box.
        ptx::tmem_wait_ld();
        ptx::tmem_wait_st();
        if (OSTAGE && lane == 0)
            ptx::bulk_wait_all();
    }

    ptx::tc_fence_before_sync();
    __syncthreads();
    if (warp == MMA_WARP) {
        ptx::tc_fence_after_sync();
        ptx::tmem_dealloc(tmem, TMEM_COLS);
    }
}

// Takes the device error word: zeroes it and leaves its old value in
// g_error_taken, in one atomic exchange, so no bit set meanwhile is lost.
__device__ unsigned int g_error_taken;
__global__ void error_word_take_kernel() { g_error_taken = atomicExch(&g_error_word, 0u); }

// Failure-detection self-test: one thread waits on a barrier nothing arrives on.
__global__ void wait_timeout_selftest_kernel(uint64_t limit_ns)
{
    __shared__ __align__(8) uint64_t barrier_word;
    __shared__ int abort_word;
    const uint32_t b = ptx::smem_u32(&barrier_word);
    if (threadIdx.x == 0) {
        ptx::mbar_init(b, 1);
        abort_word = 0;
        ptx::fence_barrier_init();
    }
    __syncthreads();
    if (threadIdx.x == 0)
        (void)wait_bounded(b, 0, &abort_word, limit_ns);
    __syncthreads();
}

}  // namespace vdx
