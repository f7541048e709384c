// Host side of libvdx: the C ABI declared in include/vdx.h.
//
// Validation happens before any CUDA call; then, once per device, the device
// is checked to be sm_103 and the kernels' shared-memory limits are raised;
// then three 3-D TMA tensor maps (head dim, sequence, batch*head) are encoded
// and one kernel is launched on the caller's stream (joint attention with
// segment ids first launches two small kernels that build its key-tile
// lists).  The device calls allocate only the workspace of the split tail and
// of the key-tile lists (per device and stream, made once, grown, kept); the
// host-buffer calls also keep their pipeline's staging slots and streams.
#include <cuda.h>
#include <cuda_runtime.h>

#include <climits>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <map>
#include <mutex>
#include <tuple>
#include <utility>
#include <vector>

#include "attn_fwd_kernel.cuh"
#include "rope3d.cuh"
#include "vdx.h"

namespace {

constexpr int kVersion = 1 * 10000 + 0 * 100 + 0;
constexpr uint64_t kWaitLimitNs = 2000000000ull;   // 2 s per in-kernel wait
constexpr int kMaxDevices = 64;
constexpr int kMinPartTiles = 8;   // key tiles a part of a cut single-round call holds at least

using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                   const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn()
{
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *ptr = nullptr;
        cudaDriverEntryPointQueryResult q{};
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(ptr);
    });
    return fn;
}

struct DeviceState {
    std::once_flag once;
    int status = VDX_OK;
    int sms = 0;   // streaming multiprocessors: one persistent CTA each
};
DeviceState g_devices[kMaxDevices];

// Kernel configurations: (Q buffers, K/V stages) per head dim.  D = 128 fits
// one Q buffer and two K/V stages (a second Q buffer would leave one stage,
// which serialises the K/V loads and measured slower even on the two-tile
// text cross-attention); D = 64 fits two Q buffers (the next item's Q loads a
// whole item ahead) and four stages.

template <int D, int MODE, int QBUF, int NSTAGE>
cudaError_t raise_smem_limit()
{
    return cudaFuncSetAttribute(vdx::attn_fwd_kernel<D, MODE, QBUF, NSTAGE>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize,
                                vdx::Layout<D, QBUF, NSTAGE, vdx::stages_out<MODE>()>::ALLOC);
}

cudaError_t raise_all_smem_limits()
{
    cudaError_t e = cudaSuccess;
    using namespace vdx;
    for (cudaError_t r : {raise_smem_limit<128, MODE_DENSE, 1, 2>(), raise_smem_limit<128, MODE_VARLEN, 1, 2>(),
                          raise_smem_limit<128, MODE_SEG, 1, 2>(), raise_smem_limit<128, MODE_WIN, 1, 2>(),
                          raise_smem_limit<64, MODE_DENSE, 2, 4>(), raise_smem_limit<64, MODE_VARLEN, 2, 4>(),
                          raise_smem_limit<64, MODE_SEG, 2, 4>(), raise_smem_limit<64, MODE_WIN, 2, 4>()})
        if (r != cudaSuccess)
            e = r;
    return e;
}

template <int D, int MODE, int QBUF, int NSTAGE>
cudaError_t launch(dim3 grid, const CUtensorMap &mq, const CUtensorMap &mk, const CUtensorMap &mv,
                   const CUtensorMap &mo, const vdx::AttnParams &p, const vdx::SegParams &sp, cudaStream_t s)
{
    vdx::attn_fwd_kernel<D, MODE, QBUF, NSTAGE>
        <<<grid, vdx::NUM_THREADS, vdx::Layout<D, QBUF, NSTAGE, vdx::stages_out<MODE>()>::ALLOC, s>>>(mq, mk, mv, mo,
                                                                                                      p, sp);
    return cudaGetLastError();
}

// One-time per-device check and kernel attribute set-up (current device).
// Returns the status and, through *sms, the device's multiprocessor count.
int device_ready(int *sms = nullptr)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess)
        return VDX_ERR_CUDA;
    if (dev < 0 || dev >= kMaxDevices)
        return VDX_ERR_UNSUPPORTED;
    DeviceState &st = g_devices[dev];
    std::call_once(st.once, [&] {
        int major = 0, minor = 0;
        if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess) {
            st.status = VDX_ERR_CUDA;
            return;
        }
        if (major != 10 || minor != 3) {
            st.status = VDX_ERR_DEVICE;
            return;
        }
        if (cudaDeviceGetAttribute(&st.sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || st.sms <= 0) {
            st.status = VDX_ERR_CUDA;
            return;
        }
        if (raise_all_smem_limits() != cudaSuccess) {
            st.status = VDX_ERR_CUDA;
            return;
        }
        st.status = encode_fn() ? VDX_OK : VDX_ERR_CUDA;
    });
    if (sms)
        *sms = st.sms;
    return st.status;
}

// Library-owned device buffers, one per (device, stream, kind): calls on one
// stream run in order, so they can share them; calls on different streams
// never do.  Allocated on the first call that needs one and kept until
// vdx_release or exit.  The split-tail scratch is allocated at its bound
// (one part per multiprocessor at D = 128), so once a stream has one no later
// dense call allocates or frees anything; the kinds that scale with the
// problem grow when a call needs more (cudaFree waits for work still using
// the old buffer).
struct Workspace {
    void *ptr = nullptr;
    size_t bytes = 0;
};
// kind: WS_SPLIT (split tail), WS_LISTS (key-tile lists of segment calls),
// WS_ROPE_K / WS_ROPE_Q (the turned K and Q of vdx_attn_fwd_rope3d).
enum { WS_SPLIT = 0, WS_LISTS = 1, WS_ROPE_K = 2, WS_ROPE_Q = 3, WS_KINDS = 4 };
std::mutex g_ws_mutex;
std::map<std::tuple<int, cudaStream_t, int>, Workspace> g_ws;

int workspace(int dev, cudaStream_t stream, size_t bytes, void **out, int kind)
{
    std::lock_guard<std::mutex> lock(g_ws_mutex);
    Workspace &w = g_ws[std::make_tuple(dev, stream, kind)];
    if (w.bytes < bytes) {
        if (w.ptr && cudaFree(w.ptr) != cudaSuccess)
            return VDX_ERR_CUDA;
        w.ptr = nullptr;
        w.bytes = 0;
        if (cudaMalloc(&w.ptr, bytes) != cudaSuccess)
            return VDX_ERR_CUDA;
        w.bytes = bytes;
    }
    *out = w.ptr;
    return VDX_OK;
}

// Frees the workspaces of (dev, stream); the caller has synchronised stream.
int release_workspaces(int dev, cudaStream_t stream)
{
    std::lock_guard<std::mutex> lock(g_ws_mutex);
    int st = VDX_OK;
    for (int kind = 0; kind < WS_KINDS; ++kind) {
        auto it = g_ws.find(std::make_tuple(dev, stream, kind));
        if (it == g_ws.end())
            continue;
        if (it->second.ptr && cudaFree(it->second.ptr) != cudaSuccess)
            st = VDX_ERR_CUDA;
        g_ws.erase(it);
    }
    return st;
}

size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Split-tail scratch of `cells` (tail units x parts, at most one per CTA)
// at head dim D: unnormalised O, then the row statistics, then the counters.
struct SplitLayout {
    size_t o_bytes, st_bytes, cnt_bytes;
    size_t total() const { return o_bytes + st_bytes + cnt_bytes; }
};
SplitLayout split_layout(size_t cells, size_t tail, int D)
{
    return {round_up(cells * 2 * vdx::BM * D * 4, 256), round_up(cells * 2 * vdx::BM * 16, 256),
            round_up(tail * 4, 256)};
}
// Its bound on a device with `sms` multiprocessors: tail x parts <= grid <= sms.
size_t split_bound_bytes(int sms) { return split_layout(sms, sms, 128).total(); }

// [B*H, rows, D] bf16 tensor as a 3-D TMA map with 64 x box_rows x 1 boxes, 128-B swizzle.
int make_map(CUtensorMap *map, const void *base, long long rows, long long bh, int D, int box_rows = vdx::BM)
{
    const cuuint64_t dims[3] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(rows),
                                static_cast<cuuint64_t>(bh)};
    const cuuint64_t strides[2] = {static_cast<cuuint64_t>(D) * 2, static_cast<cuuint64_t>(rows) * D * 2};
    const cuuint32_t box[3] = {64, static_cast<cuuint32_t>(box_rows), 1};
    const cuuint32_t estr[3] = {1, 1, 1};
    const CUresult r = encode_fn()(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base), dims, strides,
                                   box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? VDX_OK : VDX_ERR_CUDA;
}

// [B*H, F, Hp, Wp, D] bf16 tensor (a token grid per (b, h)) as a 5-D TMA map
// (D, Wp, Hp, F, B*H) with 64 x bw x bh x bt x 1 boxes: one box is a 3-D
// brick of bt*bh*bw tokens, landing as that many 128-byte rows (w fastest)
// in the 128-byte swizzle of the 3-D maps.
int make_map5(CUtensorMap *map, const void *base, const vdx::WinGrid &g, long long bh, int D, int lt, int lh, int lw)
{
    const cuuint64_t dims[5] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(g.Wp),
                                static_cast<cuuint64_t>(g.Hp), static_cast<cuuint64_t>(g.F),
                                static_cast<cuuint64_t>(bh)};
    const cuuint64_t row = static_cast<cuuint64_t>(D) * 2;
    const cuuint64_t strides[4] = {row, row * g.Wp, row * g.Wp * g.Hp, row * g.Wp * g.Hp * g.F};
    const cuuint32_t box[5] = {64, 1u << lw, 1u << lh, 1u << lt, 1};
    const cuuint32_t estr[5] = {1, 1, 1, 1, 1};
    const CUresult r = encode_fn()(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<void *>(base), dims, strides,
                                   box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? VDX_OK : VDX_ERR_CUDA;
}

// Key boxes of side 2^lk along one axis of length L, summed over the units
// along it (each covering `span` consecutive positions from span * j).
long long axis_boxes(int L, int k, int neighbourhood, int span, int lk)
{
    long long n = 0;
    for (int p0 = 0; p0 < L; p0 += span) {
        int lo, hi;
        vdx::axis_union(p0, p0 + span - 1, L, k, neighbourhood, lo, hi);
        n += (hi - lo + (1 << lk)) >> lk;
    }
    return n;
}

// Brick and key-box shapes of a windowed problem: among all query bricks of
// 128 tokens (a unit is two of them stacked in t) and all key boxes of 128
// tokens whose t-slices hold at most 32 keys, the pair with the fewest key
// steps in all, each unit also counted as two steps for its start and
// epilogue.  The step count is a product of per-axis sums, so the search is
// cheap.  Fills the shape fields of g; returns the units per (b, h).
long long choose_win_shapes(vdx::WinGrid &g)
{
    double best = -1.0;
    long long best_units = 0;
    for (int qt = 0; qt <= 7; ++qt)
        for (int qh = 0; qt + qh <= 7; ++qh) {
            const int qw = 7 - qt - qh;
            const long long nut = (g.F + (2 << qt) - 1) / (2 << qt);
            const long long nuh = (g.Hp + (1 << qh) - 1) >> qh, nuw = (g.Wp + (1 << qw) - 1) >> qw;
            const long long units = nut * nuh * nuw;
            for (int kt = 2; kt <= 7; ++kt)
                for (int kh = 0; kt + kh <= 7; ++kh) {
                    const int kw = 7 - kt - kh;
                    const double steps = static_cast<double>(axis_boxes(g.F, g.kt, g.neighbourhood, 2 << qt, kt)) *
                                         static_cast<double>(axis_boxes(g.Hp, g.kh, g.neighbourhood, 1 << qh, kh)) *
                                         static_cast<double>(axis_boxes(g.Wp, g.kw, g.neighbourhood, 1 << qw, kw));
                    const double cost = steps + 2.0 * static_cast<double>(units);
                    if (best < 0 || cost < best) {
                        best = cost;
                        best_units = units;
                        g.qlt = qt, g.qlh = qh, g.qlw = qw;
                        g.klt = kt, g.klh = kh, g.klw = kw;
                        g.nuh = static_cast<int>(nuh), g.nuw = static_cast<int>(nuw);
                    }
                }
        }
    return best_units;
}

bool aligned(const void *p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

bool overlaps(const void *a, size_t na, const void *b, size_t nb)
{
    const uintptr_t x = reinterpret_cast<uintptr_t>(a), y = reinterpret_cast<uintptr_t>(b);
    return x < y + nb && y < x + na;
}

// Per-problem-kind inputs: the valid key counts (MODE_VARLEN), the segment
// ids (MODE_SEG) or the grid and window (MODE_WIN).  Device pointers for the
// device calls; host pointers when handed to the host-buffer pipeline.
struct KeyRule {
    int mode = vdx::MODE_DENSE;
    const int *kv_lens = nullptr;
    const int *q_seg = nullptr;
    const int *kv_seg = nullptr;
    vdx::WinGrid win{};   // MODE_WIN
};

// Checks the arguments of an attention call without any CUDA call.  VDX_OK
// with *empty = true means there is nothing to launch.
int attn_check(const void *q, const void *k, const void *v, const void *out, const float *lse, int B, int H, int Sq,
               int Skv, int D, const KeyRule &rule, float scale, bool *empty)
{
    const bool varlen = rule.mode == vdx::MODE_VARLEN;
    const bool seg = rule.mode == vdx::MODE_SEG;
    const int *kv_lens = rule.kv_lens;
    *empty = false;
    if (!q || !k || !v || !out || (varlen && !kv_lens) || (seg && (!rule.q_seg || !rule.kv_seg)))
        return VDX_ERR_INVALID_ARG;
    if (B < 0 || H < 0 || Sq < 0 || Skv < 0)
        return VDX_ERR_INVALID_ARG;
    if (D != 64 && D != 128)
        return VDX_ERR_INVALID_ARG;
    if (!std::isfinite(scale))
        return VDX_ERR_INVALID_ARG;
    if (!aligned(q, 16) || !aligned(k, 16) || !aligned(v, 16) || !aligned(out, 16) || (lse && !aligned(lse, 4)) ||
        (kv_lens && !aligned(kv_lens, 4)) || (seg && (!aligned(rule.q_seg, 4) || !aligned(rule.kv_seg, 4))))
        return VDX_ERR_MISALIGNED;
    const long long bh = static_cast<long long>(B) * H;
    if (bh == 0 || Sq == 0) {
        *empty = true;
        return VDX_OK;
    }
    if (bh > INT_MAX)
        return VDX_ERR_INVALID_ARG;
    const long long q_tiles = (Sq + vdx::BM - 1) / vdx::BM;
    const long long q_pairs = (q_tiles + 1) / 2;
    if (bh * q_pairs > INT_MAX)
        return VDX_ERR_UNSUPPORTED;
    const size_t q_bytes = static_cast<size_t>(bh) * Sq * D * 2;
    const size_t kv_bytes = static_cast<size_t>(bh) * Skv * D * 2;
    if (overlaps(out, q_bytes, q, q_bytes) || (kv_bytes && (overlaps(out, q_bytes, k, kv_bytes) ||
                                                           overlaps(out, q_bytes, v, kv_bytes))))
        return VDX_ERR_INVALID_ARG;
    return VDX_OK;
}

// fixed_scratch / fixed_bytes: when set, the split-tail workspace is taken
// from that fixed device region instead of the library's allocation.
int attn_launch(const void *q, const void *k, const void *v, void *out, float *lse, int B, int H, int Sq, int Skv,
                int D, const KeyRule &rule, float scale, void *stream, void *fixed_scratch = nullptr,
                size_t fixed_bytes = 0)
{
    const bool varlen = rule.mode == vdx::MODE_VARLEN;
    const bool seg = rule.mode == vdx::MODE_SEG;
    const bool win = rule.mode == vdx::MODE_WIN;
    const int *kv_lens = rule.kv_lens;
    // ---- validation (no CUDA calls)
    bool empty = false;
    int chk = attn_check(q, k, v, out, lse, B, H, Sq, Skv, D, rule, scale, &empty);
    if (chk != VDX_OK || empty)
        return chk;
    const long long bh = static_cast<long long>(B) * H;
    const long long q_tiles = (Sq + vdx::BM - 1) / vdx::BM;
    long long q_pairs = (q_tiles + 1) / 2;
    vdx::WinGrid wg = rule.win;
    if (win) {
        // query bricks and key boxes (window_tiles.cuh); a unit is two bricks
        q_pairs = choose_win_shapes(wg);
        if (bh * q_pairs > INT_MAX)
            return VDX_ERR_UNSUPPORTED;
    }

    // ---- device set-up
    int sms = 0;
    int st = device_ready(&sms);
    if (st != VDX_OK)
        return st;

    CUtensorMap mq, mk, mv, mo;
    const long long kv_rows = Skv > 0 ? Skv : 1;   // never loaded when Skv == 0
    if (win) {
        if ((st = make_map5(&mq, q, wg, bh, D, wg.qlt, wg.qlh, wg.qlw)) != VDX_OK ||
            (st = make_map5(&mk, k, wg, bh, D, wg.klt, wg.klh, wg.klw)) != VDX_OK ||
            (st = make_map5(&mv, v, wg, bh, D, wg.klt, wg.klh, wg.klw)) != VDX_OK)
            return st;
    } else if ((st = make_map(&mq, q, Sq, bh, D)) != VDX_OK || (st = make_map(&mk, k, kv_rows, bh, D)) != VDX_OK ||
               (st = make_map(&mv, v, kv_rows, bh, D)) != VDX_OK) {
        return st;
    }
    // The output map (32-row boxes, one per softmax warp) serves the instance
    // that stores O through TMA; the others never read it.
    std::memset(&mo, 0, sizeof(mo));
    if (varlen && (st = make_map(&mo, out, Sq, bh, D, 32)) != VDX_OK)
        return st;

    vdx::AttnParams p{};
    vdx::SegParams sp{};
    p.out = static_cast<__nv_bfloat16 *>(out);
    p.lse = lse;
    p.kv_lens = kv_lens;
    p.H = H;
    p.Sq = Sq;
    p.Skv = Skv;
    p.q_pairs = static_cast<int>(q_pairs);
    p.units = static_cast<int>(bh * q_pairs);
    p.out_align32 = aligned(out, 32) ? 1 : 0;
    // A zero (or tinier than 1e-30) logit scale is raised to 1e-30: every
    // weight is then still exactly 1 for finite logits, and masked keys
    // (+-inf logits) keep weight 0 instead of inf * 0 = NaN.
    double sl2 = static_cast<double>(scale) * 1.4426950408889634074;
    if (std::fabs(sl2) < 1e-30)
        sl2 = sl2 < 0 ? -1e-30 : 1e-30;
    p.scale_log2 = static_cast<float>(sl2);
    p.wait_limit_ns = kWaitLimitNs;

    // Persistent grid: one CTA per multiprocessor (one fits per SM), each
    // taking units blockIdx.x, blockIdx.x + grid, ... so that the CTAs
    // running at any moment work on neighbouring units of the same heads.
    int G = p.units < sms ? p.units : sms;
    cudaStream_t s = static_cast<cudaStream_t>(stream);

    // Short last round: when at most half the CTAs would get a unit in it,
    // cut each of those units along the keys into parts, one per CTA, and
    // merge the parts (dense problems; varlen units vary in length).  A
    // dense call of at most half as many units as multiprocessors has only
    // such a round: its units are cut the same way, onto units x parts CTAs,
    // each part at least kMinPartTiles key tiles (shorter parts measured
    // slower than no cut: the merge outweighs them).
    const int n_kv = (Skv + vdx::BN - 1) / vdx::BN;
    int full_rounds = p.units / G;
    int tail = p.units - full_rounds * G;
    int parts = 0;
    if (rule.mode == vdx::MODE_DENSE && p.units > 0 && 2 * p.units <= sms) {
        full_rounds = 0;
        tail = p.units;
        parts = sms / tail;
        if (parts > n_kv / kMinPartTiles)
            parts = n_kv / kMinPartTiles;
    } else if (rule.mode == vdx::MODE_DENSE && full_rounds >= 1 && tail > 0) {
        parts = G / tail;
    }
    if (parts > n_kv)
        parts = n_kv;
    if (parts >= 2) {
        const SplitLayout sl = split_layout(static_cast<size_t>(tail) * parts, tail, D);
        int dev = 0;
        void *ws = nullptr;
        if (fixed_scratch) {
            if (sl.total() > fixed_bytes)
                return VDX_ERR_UNSUPPORTED;
            ws = fixed_scratch;
        } else {
            if (cudaGetDevice(&dev) != cudaSuccess)
                return VDX_ERR_CUDA;
            size_t need = split_bound_bytes(sms);
            need = need > sl.total() ? need : sl.total();
            if ((st = workspace(dev, s, need, &ws, WS_SPLIT)) != VDX_OK)
                return st;
        }
        p.split_parts = parts;
        p.full_rounds = full_rounds;
        p.tail_units = tail;
        if (full_rounds == 0)
            G = tail * parts;
        p.ws_o = static_cast<float *>(ws);
        p.ws_stats = reinterpret_cast<float *>(static_cast<char *>(ws) + sl.o_bytes);
        p.ws_count = reinterpret_cast<int *>(static_cast<char *>(ws) + sl.o_bytes + sl.st_bytes);
        if (cudaMemsetAsync(p.ws_count, 0, static_cast<size_t>(tail) * 4, s) != cudaSuccess)
            return VDX_ERR_CUDA;
    }
    if (seg) {
        // Key-tile lists per (sample, query-tile pair), shared by the heads.
        const int n_qt = static_cast<int>(q_tiles);
        const size_t pairs = static_cast<size_t>(B) * q_pairs;
        const size_t kr_bytes = round_up(static_cast<size_t>(B) * n_kv * 8, 256);
        const size_t qr_bytes = round_up(static_cast<size_t>(B) * n_qt * 8, 256);
        const size_t list_bytes = round_up(pairs * n_kv * 4, 256);
        const size_t cnt_bytes = round_up(pairs * 4, 256);
        if (pairs * n_kv > static_cast<size_t>(INT_MAX))
            return VDX_ERR_UNSUPPORTED;
        int dev = 0;
        void *ws = nullptr;
        if (cudaGetDevice(&dev) != cudaSuccess)
            return VDX_ERR_CUDA;
        if ((st = workspace(dev, s, kr_bytes + qr_bytes + list_bytes + cnt_bytes, &ws, WS_LISTS)) != VDX_OK)
            return st;
        char *base = static_cast<char *>(ws);
        int2 *krange = reinterpret_cast<int2 *>(base);
        int2 *qrange = reinterpret_cast<int2 *>(base + kr_bytes);
        uint32_t *tlist = reinterpret_cast<uint32_t *>(base + kr_bytes + qr_bytes);
        int *tcount = reinterpret_cast<int *>(base + kr_bytes + qr_bytes + list_bytes);
        const long long range_warps = static_cast<long long>(B) * (n_kv + n_qt);
        vdx::seg_tile_ranges_kernel<<<static_cast<unsigned>((range_warps + 7) / 8), 256, 0, s>>>(
            rule.q_seg, rule.kv_seg, B, Sq, Skv, n_qt, n_kv, qrange, krange);
        vdx::seg_tile_lists_kernel<<<static_cast<unsigned>((pairs + 7) / 8), 256, 0, s>>>(
            qrange, krange, B, static_cast<int>(q_pairs), n_qt, n_kv, tlist, tcount);
        if (cudaGetLastError() != cudaSuccess)
            return VDX_ERR_CUDA;
        sp.q_seg = rule.q_seg;
        sp.kv_seg = rule.kv_seg;
        sp.tlist = tlist;
        sp.tcount = tcount;
        sp.n_kt = n_kv;
    }
    if (win)
        sp.win = wg;   // no lists: each unit's key boxes follow from its index
    using vdx::MODE_DENSE;
    using vdx::MODE_SEG;
    using vdx::MODE_VARLEN;
    using vdx::MODE_WIN;
    const dim3 grid(static_cast<unsigned>(G));
    cudaError_t e;
    if (D == 128) {
        e = varlen ? launch<128, MODE_VARLEN, 1, 2>(grid, mq, mk, mv, mo, p, sp, s)
            : seg  ? launch<128, MODE_SEG, 1, 2>(grid, mq, mk, mv, mo, p, sp, s)
            : win  ? launch<128, MODE_WIN, 1, 2>(grid, mq, mk, mv, mo, p, sp, s)
                   : launch<128, MODE_DENSE, 1, 2>(grid, mq, mk, mv, mo, p, sp, s);
    } else {
        e = varlen ? launch<64, MODE_VARLEN, 2, 4>(grid, mq, mk, mv, mo, p, sp, s)
            : seg  ? launch<64, MODE_SEG, 2, 4>(grid, mq, mk, mv, mo, p, sp, s)
            : win  ? launch<64, MODE_WIN, 2, 4>(grid, mq, mk, mv, mo, p, sp, s)
                   : launch<64, MODE_DENSE, 2, 4>(grid, mq, mk, mv, mo, p, sp, s);
    }
    if (e == cudaErrorNoKernelImageForDevice)
        return VDX_ERR_DEVICE;
    return e == cudaSuccess ? VDX_OK : VDX_ERR_CUDA;
}

// ---------------------------------------------------------------- no-allocation variant
// Scratch for vdx_attn_fwd_noalloc: a fixed array in device memory, part of
// the library image, so every GPU that loads the library holds these 24 MiB
// until the process exits.  24 MiB covers the split-tail workspace of any
// call on a GPU with up to 152 multiprocessors (at most one part per
// multiprocessor: 152 x 2 x 128 x (4 x 128 + 16) bytes ~ 20.6 MB at D = 128).
constexpr size_t kNoAllocScratchBytes = size_t(24) << 20;
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

// In host code `g_noalloc_scratch` names a host-side stand-in, not the device
// array, so its device address is looked up once per device (that device
// current) and passed to the kernel.
struct NoAllocState {
    std::once_flag once;
    int status = VDX_OK;
    void *ptr = nullptr;
};
NoAllocState g_noalloc[kMaxDevices];

int noalloc_scratch(void **ptr)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess)
        return VDX_ERR_CUDA;
    if (dev < 0 || dev >= kMaxDevices)
        return VDX_ERR_UNSUPPORTED;
    NoAllocState &st = g_noalloc[dev];
    std::call_once(st.once, [&] {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) {
            st.status = VDX_ERR_CUDA;
            return;
        }
        st.ptr = p;
    });
    *ptr = st.ptr;
    return st.status;
}

// Window rule of vdx_attn_fwd_win3d(_host): odd window sizes >= 1, grid sides
// below 65536 (window bounds are packed in 16 bits), F*Hp*Wp within int.
int win_rule(int F, int Hp, int Wp, int kt, int kh, int kw, int neighbourhood, KeyRule *rule)
{
    if (F < 0 || Hp < 0 || Wp < 0 || kt < 1 || kh < 1 || kw < 1 || !(kt & kh & kw & 1))
        return VDX_ERR_INVALID_ARG;
    const long long S = static_cast<long long>(F) * Hp * Wp;
    if (S > INT_MAX || F > 65535 || Hp > 65535 || Wp > 65535)
        return VDX_ERR_UNSUPPORTED;
    rule->mode = vdx::MODE_WIN;
    rule->win.F = F;
    rule->win.Hp = Hp;
    rule->win.Wp = Wp;
    rule->win.kt = kt;
    rule->win.kh = kh;
    rule->win.kw = kw;
    rule->win.neighbourhood = neighbourhood ? 1 : 0;
    return VDX_OK;
}

int rope_launch(const vdx::RopeParams &p, bool interleaved, cudaStream_t s);   // the 3D RoPE, below

// ---------------------------------------------------------------- host-buffer pipeline
// vdx_attn_fwd_host cuts the (b, h) rows into chunks.  Chunk i is copied in
// on one stream, run on one of two compute streams (alternating, so that
// chunk i+1's CTAs take the multiprocessors that chunk i's last short round
// leaves idle) and copied out on a third.  kHostSlots device slots (inputs
// and outputs of one chunk each) rotate over the chunks; events order the
// reuse of a slot.  One pipeline per (device, caller stream), made by its
// first call, grown when a call needs larger slots (the old slots are freed,
// which waits for the device), kept until exit.
constexpr int kHostSlots = 3;

struct HostPipe {
    std::mutex mutex;   // one call at a time enqueues on a pipeline
    bool ready = false;
    cudaStream_t up = nullptr, down = nullptr, run[2] = {};
    cudaEvent_t start = nullptr, h2d[kHostSlots] = {}, comp[kHostSlots] = {}, d2h[kHostSlots] = {};
    void *buf = nullptr;
    size_t bytes = 0;
};
std::mutex g_pipes_mutex;
std::map<std::pair<int, cudaStream_t>, HostPipe> g_pipes;

HostPipe &host_pipe(int dev, cudaStream_t s)
{
    std::lock_guard<std::mutex> lock(g_pipes_mutex);
    return g_pipes[{dev, s}];   // map nodes never move
}

int host_pipe_init(HostPipe &pp)
{
    if (pp.ready)
        return VDX_OK;
    if (cudaStreamCreateWithFlags(&pp.up, cudaStreamNonBlocking) != cudaSuccess ||
        cudaStreamCreateWithFlags(&pp.down, cudaStreamNonBlocking) != cudaSuccess ||
        cudaStreamCreateWithFlags(&pp.run[0], cudaStreamNonBlocking) != cudaSuccess ||
        cudaStreamCreateWithFlags(&pp.run[1], cudaStreamNonBlocking) != cudaSuccess ||
        cudaEventCreateWithFlags(&pp.start, cudaEventDisableTiming) != cudaSuccess)
        return VDX_ERR_CUDA;
    for (int i = 0; i < kHostSlots; ++i)
        if (cudaEventCreateWithFlags(&pp.h2d[i], cudaEventDisableTiming) != cudaSuccess ||
            cudaEventCreateWithFlags(&pp.comp[i], cudaEventDisableTiming) != cudaSuccess ||
            cudaEventCreateWithFlags(&pp.d2h[i], cudaEventDisableTiming) != cudaSuccess)
            return VDX_ERR_CUDA;
    pp.ready = true;
    return VDX_OK;
}

// A chunk: rows [row0, row0 + rows) of the flattened (b, h) rows, launched as
// B x H = nb x nh; its per-sample data (text lengths, segment ids) starts at
// sample b0.
struct HostChunk {
    long long row0;
    int rows, nb, nh;
    long long b0;
};

// Chunks of r rows.  With per-sample data a chunk holds heads of one sample
// (r <= H) or whole samples (r a multiple of H), so that one offset into that
// data serves a launch.
std::vector<HostChunk> make_chunks(long long r, int B, int H, bool per_sample)
{
    std::vector<HostChunk> chunks;
    const long long bh = static_cast<long long>(B) * H;
    if (!per_sample) {
        for (long long r0 = 0; r0 < bh; r0 += r) {
            const int n = static_cast<int>(bh - r0 < r ? bh - r0 : r);
            chunks.push_back({r0, n, 1, n, 0});
        }
    } else if (r <= H) {
        for (int b = 0; b < B; ++b)
            for (int h0 = 0; h0 < H; h0 += static_cast<int>(r)) {
                const int n = static_cast<int>(H - h0 < r ? H - h0 : r);
                chunks.push_back({static_cast<long long>(b) * H + h0, n, 1, n, b});
            }
    } else {
        const int per = static_cast<int>(r / H);
        for (int b0 = 0; b0 < B; b0 += per) {
            const int nb = B - b0 < per ? B - b0 : per;
            chunks.push_back({static_cast<long long>(b0) * H, nb * H, nb, H, b0});
        }
    }
    return chunks;
}

// Rounds of one launch: `units` units of equal cost on min(units, sms)
// persistent CTAs, a short last round cut along the keys into parts when the
// dense split applies (attn_launch's rule).
double launch_rounds(long long units, int sms, int n_kv, bool dense)
{
    if (dense && units > 0 && 2 * units <= sms) {   // a single round cut along the keys
        long long parts = sms / units;
        if (parts > n_kv / kMinPartTiles)
            parts = n_kv / kMinPartTiles;
        return parts >= 2 ? 1.0 / static_cast<double>(parts) : 1.0;
    }
    const long long G = units < sms ? units : sms;
    const long long full = units / G, tail = units - full * G;
    if (tail == 0)
        return static_cast<double>(full);
    long long parts = (dense && full >= 1) ? G / tail : 0;
    if (parts > n_kv)
        parts = n_kv;
    return static_cast<double>(full) + (parts >= 2 ? 1.0 / static_cast<double>(parts) : 1.0);
}

// Cost model of the pipeline, used only to choose the chunk size: the host
// link moves kLinkBps each way while both directions are busy (pinned
// memory), a copy costs kCopyS more; a multiprocessor runs the kernel at
// kSmFlops plus kUnitS per unit; a launch costs kLaunchS.
constexpr double kLinkBps = 170e9;
constexpr double kCopyS = 5e-6;
constexpr double kSmFlops = 10.2e12;
constexpr double kUnitS = 4e-6;
constexpr double kLaunchS = 5e-6;

// Modelled seconds of a call.  Chunk i's copy in follows chunk i-1's and the
// kernel of the chunk that last held its slot; its kernel starts after its
// copy in and that chunk's copy out, and -- the kernels of consecutive chunks
// overlapping -- the GPU works through it as a fluid share of all
// multiprocessors after the previous chunk, except that the last chunk's
// short round is whole; its copy out follows chunk i-1's and its kernel.
double model_seconds(const std::vector<HostChunk> &chunks, double in_row, double out_row, long long per_row,
                     double unit_s, int sms, int n_kv, bool dense)
{
    const size_t n = chunks.size();
    std::vector<double> up(n), gpu(n), down(n);
    for (size_t i = 0; i < n; ++i) {
        const double rows = chunks[i].rows;
        const long long units = chunks[i].rows * per_row;
        double t = i ? up[i - 1] : 0.0;
        if (i >= kHostSlots && gpu[i - kHostSlots] > t)
            t = gpu[i - kHostSlots];
        up[i] = t + 3 * kCopyS + rows * in_row / kLinkBps;
        double start = up[i];
        if (i >= kHostSlots && down[i - kHostSlots] > start)
            start = down[i - kHostSlots];
        const double prev = i ? gpu[i - 1] : 0.0;
        gpu[i] = (prev > start ? prev : start) + kLaunchS + static_cast<double>(units) * unit_s / sms;
        if (i + 1 == n) {
            const double whole = start + kLaunchS + launch_rounds(units, sms, n_kv, dense) * unit_s;
            gpu[i] = whole > gpu[i] ? whole : gpu[i];
        }
        t = gpu[i];
        if (i && down[i - 1] > t)
            t = down[i - 1];
        down[i] = t + 2 * kCopyS + rows * out_row / kLinkBps;
    }
    return n ? down[n - 1] : 0.0;
}

// Rows per chunk when the caller leaves it to the library: the candidate
// with the shortest modelled call (at most 64 chunks; with per-sample data,
// heads of one sample or whole samples); fewer chunks on a tie.  kv_lens
// (host, may be NULL) refines the keys a unit visits; otherwise every key
// tile counts (an upper bound for segment and window problems).
long long auto_chunk_rows(int B, int H, int Sq, int Skv, int D, const int *kv_lens, bool per_sample, bool lse,
                          int sms)
{
    const long long bh = static_cast<long long>(B) * H;
    const bool varlen = per_sample;
    const long long per_row = (static_cast<long long>(Sq) + 2 * vdx::BM - 1) / (2 * vdx::BM);
    const int n_kv = (Skv + vdx::BN - 1) / vdx::BN;
    double keys = static_cast<double>(n_kv) * vdx::BN;   // keys a unit visits (whole tiles)
    if (kv_lens) {
        double sum = 0.0;
        for (int b = 0; b < B; ++b) {
            const int L = kv_lens[b] < 0 ? 0 : (kv_lens[b] > Skv ? Skv : kv_lens[b]);
            sum += static_cast<double>((L + vdx::BN - 1) / vdx::BN) * vdx::BN;
        }
        keys = B ? sum / B : 0.0;
    }
    const double unit_s = 2.0 * vdx::BM * keys * D * 4.0 / kSmFlops + kUnitS;
    const double in_row = (static_cast<double>(Sq) + 2.0 * Skv) * D * 2.0;
    const double out_row = static_cast<double>(Sq) * D * 2.0 + (lse ? 4.0 * Sq : 0.0);
    std::vector<long long> cand;
    if (!varlen) {
        for (long long c = 1; c <= 64 && c <= bh; ++c)
            cand.push_back((bh + c - 1) / c);
    } else {
        for (int c = 1; c <= H; ++c)
            if (static_cast<long long>(B) * c <= 64)
                cand.push_back((H + c - 1) / c);
        for (int m = 2; m <= B; ++m)
            if ((B + m - 1) / m <= 64)
                cand.push_back(static_cast<long long>(m) * H);
    }
    long long best = bh;
    double best_s = model_seconds(make_chunks(bh, B, H, varlen), in_row, out_row, per_row, unit_s, sms, n_kv, !varlen);
    for (long long r : cand) {
        const double t = model_seconds(make_chunks(r, B, H, varlen), in_row, out_row, per_row, unit_s, sms, n_kv,
                                       !varlen);
        if (t < best_s * 0.999 || (t <= best_s * 1.001 && r > best)) {
            best_s = t;
            best = r;
        }
    }
    return best;
}

// The host-buffer pipeline behind vdx_attn_fwd_host and its segment and
// window variants.  hr holds HOST pointers to the per-sample data (kv_lens
// [B]; q_seg [B, Sq] and kv_seg [B, Skv]); they are copied to the device once
// per call.  Window problems share one grid, so their chunks are any rows.
int host_pipeline(const void *q, const void *k, const void *v, void *out, float *lse, int B, int H, int Sq, int Skv,
                  int D, const KeyRule &hr, float scale, long long chunk_rows, void *stream,
                  const vdx::RopeParams *rope = nullptr, bool rope_interleaved = true)
{
    // ---- validation (no CUDA calls)
    const bool varlen = hr.mode == vdx::MODE_VARLEN, seg = hr.mode == vdx::MODE_SEG;
    if (!q || !k || !v || !out || B < 0 || H < 0 || Sq < 0 || Skv < 0 || (D != 64 && D != 128) ||
        !std::isfinite(scale) || chunk_rows < 0 || (varlen && !hr.kv_lens) || (seg && (!hr.q_seg || !hr.kv_seg)))
        return VDX_ERR_INVALID_ARG;
    const long long bh = static_cast<long long>(B) * H;
    if (bh == 0 || Sq == 0)
        return VDX_OK;
    if (bh > INT_MAX || static_cast<double>(bh) * (static_cast<double>(Sq) + Skv) * D > 1e17)
        return VDX_ERR_INVALID_ARG;
    const size_t row_q = static_cast<size_t>(Sq) * D * 2, row_kv = static_cast<size_t>(Skv) * D * 2;
    const size_t row_l = static_cast<size_t>(Sq) * 4;
    const size_t q_bytes = bh * row_q, kv_bytes = bh * row_kv, l_bytes = bh * row_l;
    if (overlaps(out, q_bytes, q, q_bytes) ||
        (kv_bytes && (overlaps(out, q_bytes, k, kv_bytes) || overlaps(out, q_bytes, v, kv_bytes))) ||
        (lse && (overlaps(lse, l_bytes, out, q_bytes) || overlaps(lse, l_bytes, q, q_bytes) ||
                 (kv_bytes && (overlaps(lse, l_bytes, k, kv_bytes) || overlaps(lse, l_bytes, v, kv_bytes))))))
        return VDX_ERR_INVALID_ARG;
    const bool per_sample = varlen || seg;

    // ---- device set-up
    int sms = 0, dev = 0;
    int st = device_ready(&sms);
    if (st != VDX_OK)
        return st;
    if (cudaGetDevice(&dev) != cudaSuccess)
        return VDX_ERR_CUDA;

    // ---- chunks
    long long r = chunk_rows > 0 ? (chunk_rows < bh ? chunk_rows : bh)
                                 : auto_chunk_rows(B, H, Sq, Skv, D, hr.kv_lens, per_sample, lse != nullptr, sms);
    if (per_sample && r > H)
        r -= r % H;
    const std::vector<HostChunk> chunks = make_chunks(r, B, H, per_sample);
    long long R = 0;
    for (const HostChunk &c : chunks)
        R = c.rows > R ? c.rows : R;

    // ---- pipeline state and slots: [per-sample data] then kHostSlots x [q | k | v | out | lse]
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    HostPipe &pp = host_pipe(dev, s);
    std::lock_guard<std::mutex> lock(pp.mutex);
    if ((st = host_pipe_init(pp)) != VDX_OK)
        return st;
    const size_t qseg_b = seg ? round_up(static_cast<size_t>(B) * Sq * 4, 256) : 0;
    const size_t lens_b = varlen ? round_up(static_cast<size_t>(B) * 4, 256)
                                 : (seg ? qseg_b + round_up(static_cast<size_t>(B) * Skv * 4, 256) : 0);
    const size_t sq_b = round_up(R * row_q, 256), skv_b = round_up(R * row_kv, 256);
    const size_t sl_b = lse ? round_up(R * row_l, 256) : 0;
    const size_t slot_b = 2 * sq_b + 2 * skv_b + sl_b;
    if (pp.bytes < lens_b + kHostSlots * slot_b) {
        if (pp.buf && cudaFree(pp.buf) != cudaSuccess)
            return VDX_ERR_CUDA;
        pp.buf = nullptr;
        pp.bytes = 0;
        if (cudaMalloc(&pp.buf, lens_b + kHostSlots * slot_b) != cudaSuccess)
            return VDX_ERR_CUDA;
        pp.bytes = lens_b + kHostSlots * slot_b;
    }
    char *base = static_cast<char *>(pp.buf);
    int *d_lens = reinterpret_cast<int *>(base);                 // varlen: [B]
    int *d_qseg = reinterpret_cast<int *>(base);                 // segments: [B, Sq], then [B, Skv]
    int *d_kvseg = reinterpret_cast<int *>(base + qseg_b);
    auto slot = [&](int i, int part) {   // part: 0 q, 1 k, 2 v, 3 out, 4 lse
        const size_t off[5] = {0, sq_b, sq_b + skv_b, sq_b + 2 * skv_b, 2 * sq_b + 2 * skv_b};
        return base + lens_b + static_cast<size_t>(i) * slot_b + off[part];
    };

    // ---- enqueue: everything after the caller's earlier work on `stream`.
    // A failure after the first enqueue still makes `stream` wait for all the
    // pipeline's streams, so that no later call reuses a slot under work in
    // flight.
    auto fail = [&](int code) {
        for (cudaStream_t own : {pp.up, pp.run[0], pp.run[1], pp.down})
            if (cudaEventRecord(pp.start, own) == cudaSuccess)
                (void)cudaStreamWaitEvent(s, pp.start, 0);
        return code;
    };
    const char *qh = static_cast<const char *>(q), *kh = static_cast<const char *>(k);
    const char *vh = static_cast<const char *>(v);
    char *oh = static_cast<char *>(out), *lh = reinterpret_cast<char *>(lse);
    if (cudaEventRecord(pp.start, s) != cudaSuccess || cudaStreamWaitEvent(pp.up, pp.start, 0) != cudaSuccess ||
        cudaStreamWaitEvent(pp.run[0], pp.start, 0) != cudaSuccess ||
        cudaStreamWaitEvent(pp.run[1], pp.start, 0) != cudaSuccess)
        return fail(VDX_ERR_CUDA);
    if (varlen && cudaMemcpyAsync(d_lens, hr.kv_lens, static_cast<size_t>(B) * 4, cudaMemcpyHostToDevice, pp.up) !=
                      cudaSuccess)
        return fail(VDX_ERR_CUDA);
    if (seg && (cudaMemcpyAsync(d_qseg, hr.q_seg, static_cast<size_t>(B) * Sq * 4, cudaMemcpyHostToDevice, pp.up) !=
                    cudaSuccess ||
                (Skv > 0 && cudaMemcpyAsync(d_kvseg, hr.kv_seg, static_cast<size_t>(B) * Skv * 4,
                                            cudaMemcpyHostToDevice, pp.up) != cudaSuccess)))
        return fail(VDX_ERR_CUDA);
    const size_t n = chunks.size();
    for (size_t i = 0; i <= n; ++i) {
        if (i < n) {
            // copy chunk i in once the slot's previous chunk has run, then run it
            // once that chunk's results are out
            const HostChunk &c = chunks[i];
            const int sl = static_cast<int>(i % kHostSlots);
            cudaStream_t rs = pp.run[i & 1];
            if (i >= kHostSlots && cudaStreamWaitEvent(pp.up, pp.comp[sl], 0) != cudaSuccess)
                return fail(VDX_ERR_CUDA);
            const size_t nq = c.rows * row_q, nkv = c.rows * row_kv;
            if (cudaMemcpyAsync(slot(sl, 0), qh + c.row0 * row_q, nq, cudaMemcpyHostToDevice, pp.up) != cudaSuccess ||
                (nkv && (cudaMemcpyAsync(slot(sl, 1), kh + c.row0 * row_kv, nkv, cudaMemcpyHostToDevice, pp.up) !=
                             cudaSuccess ||
                         cudaMemcpyAsync(slot(sl, 2), vh + c.row0 * row_kv, nkv, cudaMemcpyHostToDevice, pp.up) !=
                             cudaSuccess)) ||
                cudaEventRecord(pp.h2d[sl], pp.up) != cudaSuccess ||
                cudaStreamWaitEvent(rs, pp.h2d[sl], 0) != cudaSuccess ||
                (i >= kHostSlots && cudaStreamWaitEvent(rs, pp.d2h[sl], 0) != cudaSuccess))
                return fail(VDX_ERR_CUDA);
            if (rope) {
                // the 3D RoPE of the chunk's q and k, in place in the slot (row by row,
                // so a chunk of rows turns exactly as the whole tensor would)
                vdx::RopeParams rq = *rope;
                rq.BH = c.rows;
                rq.copy_all = 0;
                rq.S = Sq;
                rq.x = rq.y = reinterpret_cast<__nv_bfloat16 *>(slot(sl, 0));
                vdx::RopeParams rk = rq;
                rk.S = Skv;
                rk.x = rk.y = reinterpret_cast<__nv_bfloat16 *>(slot(sl, 1));
                if ((st = rope_launch(rq, rope_interleaved, rs)) != VDX_OK ||
                    (st = rope_launch(rk, rope_interleaved, rs)) != VDX_OK)
                    return fail(st);
            }
            KeyRule rule = hr;   // window problems: the grid as given
            if (varlen)
                rule.kv_lens = d_lens + c.b0;
            if (seg) {
                rule.q_seg = d_qseg + c.b0 * Sq;
                rule.kv_seg = d_kvseg + c.b0 * Skv;
            }
            st = attn_launch(slot(sl, 0), slot(sl, 1), slot(sl, 2), slot(sl, 3),
                             lse ? reinterpret_cast<float *>(slot(sl, 4)) : nullptr, c.nb, c.nh, Sq, Skv, D, rule,
                             scale, rs);
            if (st != VDX_OK)
                return fail(st);
            if (cudaEventRecord(pp.comp[sl], rs) != cudaSuccess)
                return fail(VDX_ERR_CUDA);
        }
        if (i >= 1) {
            // copy chunk i-1 out once its kernel is done
            const HostChunk &c = chunks[i - 1];
            const int sl = static_cast<int>((i - 1) % kHostSlots);
            if (cudaStreamWaitEvent(pp.down, pp.comp[sl], 0) != cudaSuccess ||
                cudaMemcpyAsync(oh + c.row0 * row_q, slot(sl, 3), c.rows * row_q, cudaMemcpyDeviceToHost, pp.down) !=
                    cudaSuccess ||
                (lse && cudaMemcpyAsync(lh + c.row0 * row_l, slot(sl, 4), c.rows * row_l, cudaMemcpyDeviceToHost,
                                        pp.down) != cudaSuccess) ||
                cudaEventRecord(pp.d2h[sl], pp.down) != cudaSuccess)
                return fail(VDX_ERR_CUDA);
        }
    }
    // the caller's stream resumes once the last result is on the host
    if (cudaStreamWaitEvent(s, pp.d2h[(n - 1) % kHostSlots], 0) != cudaSuccess)
        return fail(VDX_ERR_CUDA);
    return VDX_OK;
}

// The rotation's grid, head-dim split and base, pointers aside.
bool rope_dims_ok(int D, int F, int Hp, int Wp, int s0, int d_t, int d_h, int d_w, float theta)
{
    return F >= 0 && Hp >= 0 && Wp >= 0 && s0 >= 0 && D >= 2 && D <= 512 && !(D & 1) && d_t >= 0 && d_h >= 0 &&
           d_w >= 0 && !((d_t | d_h | d_w) & 1) && static_cast<long long>(d_t) + d_h + d_w <= D &&
           std::isfinite(theta) && theta > 0.f;
}

// Checks the arguments of a rotation (no CUDA calls) and fills p (p->BH == 0
// or S == 0: nothing to do).
int rope_args(const void *x, const void *y, int B, int H, int S, int D, int F, int Hp, int Wp, int s0, int d_t,
              int d_h, int d_w, float theta, vdx::RopeParams *out_p)
{
    *out_p = vdx::RopeParams{};
    if (!x || !y || B < 0 || H < 0 || S < 0 || !rope_dims_ok(D, F, Hp, Wp, s0, d_t, d_h, d_w, theta))
        return VDX_ERR_INVALID_ARG;
    if (!aligned(x, 4) || !aligned(y, 4))
        return VDX_ERR_MISALIGNED;
    const long long bh = static_cast<long long>(B) * H;
    if (bh > INT_MAX)
        return VDX_ERR_INVALID_ARG;
    const size_t bytes = static_cast<size_t>(bh) * S * D * 2;
    if (x != y && overlaps(x, bytes, y, bytes))
        return VDX_ERR_INVALID_ARG;
    vdx::RopeParams p{};
    p.x = static_cast<const __nv_bfloat16 *>(x);
    p.y = static_cast<__nv_bfloat16 *>(const_cast<void *>(y));
    p.BH = static_cast<int>(bh);
    p.S = S;
    p.D = D;
    p.F = F;
    p.Hp = Hp;
    p.Wp = Wp;
    p.s0 = s0;
    p.d_t = d_t;
    p.d_h = d_h;
    p.d_w = d_w;
    p.log2_theta = static_cast<float>(std::log2(static_cast<double>(theta)));
    p.copy_all = x != y;
    *out_p = p;
    return VDX_OK;
}

// Launches the rotation p describes (validated by rope_args).
int rope_launch(const vdx::RopeParams &p, bool interleaved, cudaStream_t s)
{
    int sms = 0;
    const int st = device_ready(&sms);
    if (st != VDX_OK)
        return st;
    const int D = p.D, S = p.S;
    const void *x = p.x, *y = p.y;
    if (interleaved && D % 8 == 0 && aligned(x, 16) && aligned(y, 16)) {
        // 16-byte chunks: four pairs per thread
        const int chunks = D / 8;
        const int tok = 256 / chunks;
        const long long groups = (S + tok - 1) / tok;
        const long long cap = static_cast<long long>(sms) * vdx::ROPE_VEC_BLOCKS_PER_SM;
        const unsigned nb = static_cast<unsigned>(groups < cap ? groups : cap);
        vdx::rope3d_vec_kernel<<<dim3(nb), dim3(static_cast<unsigned>(chunks), static_cast<unsigned>(tok)), 0, s>>>(p);
    } else {
        const int pairs = D / 2;
        const int tok = 256 / pairs;
        const dim3 block(static_cast<unsigned>(pairs), static_cast<unsigned>(tok));
        const dim3 grid(static_cast<unsigned>((S + tok - 1) / tok));
        if (interleaved)
            vdx::rope3d_kernel<true><<<grid, block, 0, s>>>(p);
        else
            vdx::rope3d_kernel<false><<<grid, block, 0, s>>>(p);
    }
    return cudaGetLastError() == cudaSuccess ? VDX_OK : VDX_ERR_CUDA;
}

}  // namespace

extern "C" {

int vdx_attn_fwd_noalloc(const void *q, const void *k, const void *v, void *out, float *lse, int B, int H, int Sq,
                         int Skv, int D, float scale, void *stream)
{
    // The argument checks of vdx_attn_fwd come first, so that a bad call
    // returns the same status and touches no CUDA state; then the fixed
    // scratch's device address.
    bool empty = false;
    const int chk = attn_check(q, k, v, out, lse, B, H, Sq, Skv, D, KeyRule{}, scale, &empty);
    if (chk != VDX_OK || empty)
        return chk;
    void *scratch = nullptr;
    const int st = noalloc_scratch(&scratch);
    if (st != VDX_OK)
        return st;
    return attn_launch(q, k, v, out, lse, B, H, Sq, Skv, D, KeyRule{}, scale, stream, scratch,
                       kNoAllocScratchBytes);
}

int vdx_attn_fwd(const void *q, const void *k, const void *v, void *out, float *lse, int B, int H, int Sq, int Skv,
                 int D, float scale, void *stream)
{
    return attn_launch(q, k, v, out, lse, B, H, Sq, Skv, D, KeyRule{}, scale, stream);
}

int vdx_attn_fwd_varlen(const void *q, const void *k, const void *v, void *out, float *lse, int B, int H, int Sq,
                        int Skv_max, int D, const int *kv_lens, float scale, void *stream)
{
    KeyRule rule;
    rule.mode = vdx::MODE_VARLEN;
    rule.kv_lens = kv_lens;
    return attn_launch(q, k, v, out, lse, B, H, Sq, Skv_max, D, rule, scale, stream);
}

int vdx_attn_fwd_host(const void *q, const void *k, const void *v, void *out, float *lse, int B, int H, int Sq,
                      int Skv, int D, const int *kv_lens, float scale, long long chunk_rows, void *stream)
{
    KeyRule rule;
    if (kv_lens) {
        rule.mode = vdx::MODE_VARLEN;
        rule.kv_lens = kv_lens;
    }
    return host_pipeline(q, k, v, out, lse, B, H, Sq, Skv, D, rule, scale, chunk_rows, stream);
}

int vdx_attn_fwd_rope3d_host(const void *q, const void *k, const void *v, void *out, float *lse, int B, int H, int S,
                             int D, int F, int Hp, int Wp, int s0, int d_t, int d_h, int d_w, float theta,
                             int interleaved, float scale, long long chunk_rows, void *stream)
{
    if (!rope_dims_ok(D, F, Hp, Wp, s0, d_t, d_h, d_w, theta))
        return VDX_ERR_INVALID_ARG;
    vdx::RopeParams rp{};
    rp.D = D;
    rp.F = F;
    rp.Hp = Hp;
    rp.Wp = Wp;
    rp.s0 = s0;
    rp.d_t = d_t;
    rp.d_h = d_h;
    rp.d_w = d_w;
    rp.log2_theta = static_cast<float>(std::log2(static_cast<double>(theta)));
    return host_pipeline(q, k, v, out, lse, B, H, S, S, D, KeyRule{}, scale, chunk_rows, stream, &rp,
                         interleaved != 0);
}

int vdx_attn_fwd_segments_host(const void *q, const void *k, const void *v, void *out, float *lse, int B, int H,
                               int Sq, int Skv, int D, const int *q_seg, const int *kv_seg, float scale,
                               long long chunk_rows, void *stream)
{
    KeyRule rule;
    rule.mode = vdx::MODE_SEG;
    rule.q_seg = q_seg;
    rule.kv_seg = kv_seg;
    return host_pipeline(q, k, v, out, lse, B, H, Sq, Skv, D, rule, scale, chunk_rows, stream);
}

int vdx_attn_fwd_win3d_host(const void *q, const void *k, const void *v, void *out, float *lse, int B, int H, int F,
                            int Hp, int Wp, int D, int kt, int kh, int kw, int neighbourhood, float scale,
                            long long chunk_rows, void *stream)
{
    KeyRule rule;
    const int st = win_rule(F, Hp, Wp, kt, kh, kw, neighbourhood, &rule);
    if (st != VDX_OK)
        return st;
    const int S = F * Hp * Wp;
    return host_pipeline(q, k, v, out, lse, B, H, S, S, D, rule, scale, chunk_rows, stream);
}


int vdx_attn_fwd_win3d(const void *q, const void *k, const void *v, void *out, float *lse, int B, int H, int F,
                       int Hp, int Wp, int D, int kt, int kh, int kw, int neighbourhood, float scale, void *stream)
{
    KeyRule rule;
    const int st = win_rule(F, Hp, Wp, kt, kh, kw, neighbourhood, &rule);
    if (st != VDX_OK)
        return st;
    const int S = F * Hp * Wp;
    return attn_launch(q, k, v, out, lse, B, H, S, S, D, rule, scale, stream);
}

int vdx_rope3d(const void *x, void *y, int B, int H, int S, int D, int F, int Hp, int Wp, int s0, int d_t, int d_h,
               int d_w, float theta, int interleaved, void *stream)
{
    vdx::RopeParams p{};
    const int st = rope_args(x, y, B, H, S, D, F, Hp, Wp, s0, d_t, d_h, d_w, theta, &p);
    if (st != VDX_OK || p.BH == 0 || S == 0)
        return st;
    return rope_launch(p, interleaved != 0, static_cast<cudaStream_t>(stream));
}

int vdx_attn_fwd_rope3d(const void *q, const void *k, const void *v, void *out, float *lse, int B, int H, int S,
                        int D, int F, int Hp, int Wp, int s0, int d_t, int d_h, int d_w, float theta,
                        int interleaved, float scale, void *stream)
{
    // ---- validation: the rotation's and the attention's (no CUDA calls)
    vdx::RopeParams rq{}, rk{};
    int st = rope_args(q, q, B, H, S, D, F, Hp, Wp, s0, d_t, d_h, d_w, theta, &rq);
    if (st != VDX_OK)
        return st;
    if ((st = rope_args(k, k, B, H, S, D, F, Hp, Wp, s0, d_t, d_h, d_w, theta, &rk)) != VDX_OK)
        return st;
    if (!v || !out || !std::isfinite(scale) || (D != 64 && D != 128))
        return VDX_ERR_INVALID_ARG;
    if (!aligned(q, 16) || !aligned(k, 16) || !aligned(v, 16) || !aligned(out, 16) || (lse && !aligned(lse, 4)))
        return VDX_ERR_MISALIGNED;
    const size_t bytes = static_cast<size_t>(rk.BH) * S * D * 2;
    if (rk.BH == 0 || S == 0)
        return VDX_OK;
    if (overlaps(out, bytes, q, bytes) || overlaps(out, bytes, k, bytes) || overlaps(out, bytes, v, bytes))
        return VDX_ERR_INVALID_ARG;

    // ---- Q and K turned by the RoPE kernel into the library's per-stream
    // buffers, then the dense attention on them
    int sms = 0, dev = 0;
    if ((st = device_ready(&sms)) != VDX_OK)
        return st;
    if (cudaGetDevice(&dev) != cudaSuccess)
        return VDX_ERR_CUDA;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    void *q_rot = nullptr, *k_rot = nullptr;
    if ((st = workspace(dev, s, bytes, &q_rot, WS_ROPE_Q)) != VDX_OK ||
        (st = workspace(dev, s, bytes, &k_rot, WS_ROPE_K)) != VDX_OK)
        return st;
    rq.y = static_cast<__nv_bfloat16 *>(q_rot);
    rq.copy_all = 1;
    rk.y = static_cast<__nv_bfloat16 *>(k_rot);
    rk.copy_all = 1;
    if ((st = rope_launch(rq, interleaved != 0, s)) != VDX_OK || (st = rope_launch(rk, interleaved != 0, s)) != VDX_OK)
        return st;
    return attn_launch(q_rot, k_rot, v, out, lse, B, H, S, S, D, KeyRule{}, scale, stream);
}

int vdx_attn_fwd_segments(const void *q, const void *k, const void *v, void *out, float *lse, int B, int H, int Sq,
                          int Skv, int D, const int *q_seg, const int *kv_seg, float scale, void *stream)
{
    KeyRule rule;
    rule.mode = vdx::MODE_SEG;
    rule.q_seg = q_seg;
    rule.kv_seg = kv_seg;
    return attn_launch(q, k, v, out, lse, B, H, Sq, Skv, D, rule, scale, stream);
}

const char *vdx_status_string(int status)
{
    switch (status) {
    case VDX_OK: return "VDX_OK";
    case VDX_ERR_INVALID_ARG: return "VDX_ERR_INVALID_ARG: invalid argument";
    case VDX_ERR_UNSUPPORTED: return "VDX_ERR_UNSUPPORTED: shape not supported";
    case VDX_ERR_MISALIGNED: return "VDX_ERR_MISALIGNED: pointer alignment";
    case VDX_ERR_CUDA: return "VDX_ERR_CUDA: CUDA call failed";
    case VDX_ERR_DEVICE: return "VDX_ERR_DEVICE: current device is not sm_103";
    case VDX_ERR_TIMEOUT: return "VDX_ERR_TIMEOUT: bounded in-kernel wait expired";
    case VDX_ERR_DRAIN:
        return "VDX_ERR_DRAIN: a kernel that gave up could not confirm its copies or tensor-core work had finished";
    default: return "unknown vdx status";
    }
}

int vdx_check_device_error(void *stream)
{
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (cudaStreamSynchronize(s) != cudaSuccess)
        return VDX_ERR_CUDA;
    const int st = device_ready();
    if (st != VDX_OK)
        return st;
    // One check at a time takes the word (through one snapshot variable).
    static std::mutex take_mutex;
    std::lock_guard<std::mutex> lock(take_mutex);
    unsigned int word = 0;
    vdx::error_word_take_kernel<<<1, 1, 0, s>>>();
    if (cudaGetLastError() != cudaSuccess ||
        cudaMemcpyFromSymbolAsync(&word, vdx::g_error_taken, sizeof word, 0, cudaMemcpyDeviceToHost, s) !=
            cudaSuccess ||
        cudaStreamSynchronize(s) != cudaSuccess)
        return VDX_ERR_CUDA;
    if (word & (vdx::ERR_MMA_DRAIN | vdx::ERR_LOADS_IN_FLIGHT))
        return VDX_ERR_DRAIN;
    return word ? VDX_ERR_TIMEOUT : VDX_OK;
}

int vdx_release(void *stream)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess)
        return VDX_ERR_CUDA;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (cudaStreamSynchronize(s) != cudaSuccess)
        return VDX_ERR_CUDA;
    int st = release_workspaces(dev, s);
    // The host-buffer pipeline of (dev, stream): its slots, events, streams,
    // and the workspaces of its compute streams.
    std::unique_lock<std::mutex> lock(g_pipes_mutex);
    auto it = g_pipes.find({dev, s});
    if (it == g_pipes.end())
        return st;
    HostPipe &pp = it->second;
    {
        std::lock_guard<std::mutex> pipe_lock(pp.mutex);
        if (pp.ready) {
            for (cudaStream_t own : {pp.up, pp.run[0], pp.run[1], pp.down})
                if (cudaStreamSynchronize(own) != cudaSuccess)
                    st = VDX_ERR_CUDA;
            for (cudaStream_t own : {pp.run[0], pp.run[1]})
                if (release_workspaces(dev, own) != VDX_OK)
                    st = VDX_ERR_CUDA;
        }
        if (pp.buf && cudaFree(pp.buf) != cudaSuccess)
            st = VDX_ERR_CUDA;
        for (int i = 0; i < kHostSlots; ++i)
            for (cudaEvent_t e : {pp.h2d[i], pp.comp[i], pp.d2h[i]})
                if (e && cudaEventDestroy(e) != cudaSuccess)
                    st = VDX_ERR_CUDA;
        if (pp.start && cudaEventDestroy(pp.start) != cudaSuccess)
            st = VDX_ERR_CUDA;
        for (cudaStream_t own : {pp.up, pp.run[0], pp.run[1], pp.down})
            if (own && cudaStreamDestroy(own) != cudaSuccess)
                st = VDX_ERR_CUDA;
    }
    g_pipes.erase(it);
    return st;
}

int vdx_selftest_wait_timeout(int limit_us, void *stream)
{
    if (limit_us < 1 || limit_us > 10000000)
        return VDX_ERR_INVALID_ARG;
    const int st = device_ready();
    if (st != VDX_OK)
        return st;
    vdx::wait_timeout_selftest_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(
        static_cast<uint64_t>(limit_us) * 1000ull);
    return cudaGetLastError() == cudaSuccess ? VDX_OK : VDX_ERR_CUDA;
}

int vdx_version(void) { return kVersion; }

}  // extern "C"
