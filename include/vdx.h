/*
 * vdx.h -- C ABI of the GB300 (sm_103a) softmax attention forward library.
 *
 * The operation is the attention step of video diffusion-transformer
 * inference described in the vidax paper (arXiv 2609.18077):
 *   - Sec. 2, "3D RoPE, 3D VAEs, and flash attention": unmasked multi-head
 *     attention over patchified spatiotemporal tokens, computed with a
 *     flash-attention kernel so the Sq x Skv score matrix is never stored;
 *   - Sec. 1: patchified video volumes give tens of thousands of tokens per
 *     sample, so attention cost is quadratic in the token count;
 *   - appendix Table 4 (porting-bug taxonomy): padded text tokens must be
 *     excluded, by skipping invalid key blocks rather than by a dense
 *     (B, H, Sq, Sk) mask -- the varlen entry point below, and its
 *     generalisation to per-token segment ids for joint text-video
 *     attention (HunyuanVideo-1.5 in that entry; the ~45k-token CogVideoX1.5
 *     joint sequence of Table 3) -- vdx_attn_fwd_segments.
 *
 * For each batch b, head h and query row i, over its valid keys j (the first
 * L of them, or those of its segment):
 *     s_j  = scale * <q[b,h,i,:], k[b,h,j,:]>
 *     out[b,h,i,:] = sum_j softmax(s)_j * v[b,h,j,:]
 *     lse[b,h,i]   = ln(sum_j exp(s_j))                  (natural log)
 * No valid key gives out = 0 and lse = -inf.
 *
 * Conventions shared by every entry point:
 *   - Tensors are contiguous, row-major, bf16 (IEEE bfloat16 bits):
 *       q, out: [B, H, Sq, D];  k, v: [B, H, Skv, D];  lse: fp32 [B, H, Sq].
 *   - All tensor pointers are DEVICE pointers owned by the caller; the
 *     library never frees or keeps them after the call returns.
 *   - Memory: when the last round of work units would leave most
 *     multiprocessors idle (dense calls only; a call of at most half as many
 *     units as multiprocessors is all such a round, cut into parts of at
 *     least 8 key tiles), the library splits those units
 *     along the keys and merges the parts through a device scratch of at most
 *     (multiprocessors x 2 x 128 x (D + 4)) fp32 values plus counters -- about
 *     20.6 MB on a 152-SM GB300.  It is allocated at that bound by the first
 *     call on a stream that splits, so no later dense call on that stream
 *     allocates or frees device memory.  Segment and window calls keep their
 *     key-tile lists in a second buffer that grows with the problem
 *     (B x ceil(Sq/256) x ceil(Skv/128) x 4 bytes plus ranges, about 0.5 MB
 *     for B=2, S=45106); growing it frees the old one, which waits for the
 *     device.  These buffers belong to the library, one set per (device,
 *     stream): calls on the same stream share them in stream order, calls on
 *     different streams never share them.  They are kept until
 *     vdx_release(stream) or process exit.
 *   - q, k, v and out must be 16-byte aligned (TMA and vector stores); lse
 *     4-byte aligned.  out must not overlap q, k or v.
 *   - D must be 64 or 128.  B, H, Sq, Skv >= 0; B*H*Sq == 0 is a no-op.
 *   - The call is asynchronous on `stream` (a cudaStream_t, NULL = the legacy
 *     default stream) of the CURRENT device, which must be an sm_103 GPU.
 *   - Arguments are validated before any CUDA work; a failing call returns a
 *     vdx_status and launches nothing.  Nothing is thrown across the ABI and
 *     the library never exits the process.
 *   - Thread-safe: one-time per-device set-up is guarded internally.
 */
#ifndef VDX_H
#define VDX_H

#ifdef __cplusplus
extern "C" {
#endif

typedef enum vdx_status {
    VDX_OK = 0,
    VDX_ERR_INVALID_ARG = 1, /* null pointer, negative size, bad D, size overflow */
    VDX_ERR_UNSUPPORTED = 2, /* a shape outside what the kernel implements */
    VDX_ERR_MISALIGNED = 3,  /* a pointer breaks the alignment rules above */
    VDX_ERR_CUDA = 4,        /* a CUDA runtime/driver call failed */
    VDX_ERR_DEVICE = 5,      /* the current device is not an sm_103 GPU */
    VDX_ERR_TIMEOUT = 6,     /* a bounded in-kernel wait expired (see vdx_check_device_error) */
    VDX_ERR_DRAIN = 7        /* a kernel that gave up could not confirm that its TMA loads or
                                tensor-core operations had finished before it exited (see
                                vdx_check_device_error); treat device memory as suspect */
} vdx_status;

/*
 * Dense (non-causal, unmasked) attention forward, Sec. 2 of the paper.
 *   q   : bf16 [B,H,Sq,D]          k, v : bf16 [B,H,Skv,D]
 *   out : bf16 [B,H,Sq,D] written   lse  : fp32 [B,H,Sq] written, or NULL to skip
 *   scale: logit multiplier (1/sqrt(D) for standard attention); any finite value.
 * Skv == 0 writes out = 0 and lse = -inf.
 */
int vdx_attn_fwd(const void *q, const void *k, const void *v, void *out, float *lse,
                 int B, int H, int Sq, int Skv, int D, float scale, void *stream);

/*
 * Cross-attention to padded text tokens (appendix Table 4: per-sample valid
 * key counts instead of a dense mask).  As vdx_attn_fwd with Skv = Skv_max,
 * except that sample b attends only to keys j < clamp(kv_lens[b], 0, Skv_max).
 *   kv_lens: DEVICE int32 [B], caller-owned.  Key/value rows past a sample's
 *            length are never used and may hold any bits, NaN included.
 * Key tiles entirely past a sample's length are skipped, not masked.
 */
int vdx_attn_fwd_varlen(const void *q, const void *k, const void *v, void *out, float *lse,
                        int B, int H, int Sq, int Skv_max, int D, const int *kv_lens,
                        float scale, void *stream);

/*
 * Joint attention with segment ids (appendix Table 4: padded text tokens in
 * a joint text-video sequence are masked through segment ids so that the
 * kernel skips invalid key blocks).  As vdx_attn_fwd, except that query i of
 * sample b attends exactly the keys j with kv_seg[b*Skv + j] == q_seg[b*Sq + i].
 *   q_seg : DEVICE int32 [B, Sq],  kv_seg : DEVICE int32 [B, Skv], caller-owned,
 *           4-byte aligned, shared by all heads; any int32 values.
 * A query whose segment owns no key gets out = 0 and lse = -inf.  Key tiles
 * (128 keys) holding no id of a query tile pair's range are skipped; tiles
 * holding one id equal to the query tile's single id run unmasked; the rest
 * compare ids element by element.  Every V row must be finite: a key of
 * another segment inside a visited tile enters the tensor-core product with
 * weight exactly 0, and 0 x NaN = NaN (K may hold any bits there).
 * Two small kernels build the key-tile lists before the attention kernel, on
 * the same stream, in the library's per-stream workspace (see Memory above).
 */
int vdx_attn_fwd_segments(const void *q, const void *k, const void *v, void *out, float *lse,
                          int B, int H, int Sq, int Skv, int D, const int *q_seg, const int *kv_seg,
                          float scale, void *stream);

/*
 * Windowed 3D attention (appendix Table 4: the LTX-2.5 VAE decoder's 3D
 * neighbourhood attention, an 11 x 11 x 11 window).  As vdx_attn_fwd with
 * Sq = Skv = S = F*Hp*Wp, the tokens of each sequence being a (t, h, w) grid
 * in raster order, except that a query attends only the keys inside its
 * window.  Along an axis of length L with odd window size k (kt, kh, kw), the
 * window of position p is
 *   neighbourhood = 1: [lo, min(lo + k, L) - 1], lo = clamp(p - k/2, 0, max(L - k, 0))
 *                      (shifted inward at the border: always min(k, L) positions);
 *   neighbourhood = 0: [max(p - k/2, 0), min(p + k/2, L - 1)] (truncated).
 * Query tiles are 3-D bricks of 128 tokens and key tiles 3-D boxes of 128
 * tokens laid over the union of each unit's windows (shapes chosen per grid
 * by the library); keys outside every window of a unit are never visited,
 * and the rest compare positions element by element.  One kernel launch, no
 * workspace.  Grid sides up to 65535; VDX_ERR_UNSUPPORTED beyond.
 */
int vdx_attn_fwd_win3d(const void *q, const void *k, const void *v, void *out, float *lse,
                       int B, int H, int F, int Hp, int Wp, int D, int kt, int kh, int kw,
                       int neighbourhood, float scale, void *stream);

/*
 * 3D rotary position embedding of queries or keys (Sec. 2: each model family
 * keeps its own 3D RoPE convention over time, height and width; this call
 * takes the conventions as parameters).  The standard rotary embedding over a
 * token grid:
 *   x, y : bf16 [B, H, S, D], DEVICE pointers, caller-owned, 4-byte aligned;
 *          y == x rotates in place, otherwise the two must not overlap.
 *   F, Hp, Wp, s0 : tokens [s0, s0 + F*Hp*Wp) of each sequence are the video
 *          grid, in raster order (t, h, w); other tokens are copied unchanged.
 *   d_t, d_h, d_w : even numbers of head dims turned by t, h and w, taken in
 *          that order from dim 0; d_t + d_h + d_w <= D; the rest are copied.
 *   theta : frequency base (> 0).  Pair i of an axis part of d_a dims turns by
 *          pos * theta^(-2i/d_a):  (y_a, y_b) = (x_a cos - x_b sin, x_a sin + x_b cos).
 *   interleaved : 1: pairs (2i, 2i+1) of the part; 0: pairs (i, i + d_a/2).
 * D must be even, 2 .. 512.  Arithmetic in fp32, y rounded to bf16 (nearest
 * even).  Asynchronous on `stream`; allocates nothing.
 */
int vdx_rope3d(const void *x, void *y, int B, int H, int S, int D, int F, int Hp, int Wp, int s0,
               int d_t, int d_h, int d_w, float theta, int interleaved, void *stream);

/*
 * Self-attention with the 3D rotary embedding applied to q and k (Sec. 2:
 * each family's 3D RoPE before its flash attention): exactly
 *   vdx_rope3d(q -> q'), vdx_rope3d(k -> k'), vdx_attn_fwd(q', k', v)
 * with Sq = Skv = S and the RoPE arguments of vdx_rope3d, so the results are
 * bit for bit those of these three calls; q and k are not modified.  q' and
 * k' live in two library buffers of B*H*S*D bf16 each per (device, stream),
 * allocated by the first call, grown when needed, kept until exit; plus
 * vdx_attn_fwd's workspace.  (K cannot be turned inside the attention: every
 * query unit of a head reads all of K.  Turning each Q tile in shared memory
 * after it lands was measured 0.9 % slower per call than the separate pass.)
 * Arguments and errors as vdx_rope3d and vdx_attn_fwd together (D 64 or 128;
 * q, k, v, out 16-byte aligned).
 */
int vdx_attn_fwd_rope3d(const void *q, const void *k, const void *v, void *out, float *lse,
                        int B, int H, int S, int D, int F, int Hp, int Wp, int s0,
                        int d_t, int d_h, int d_w, float theta, int interleaved,
                        float scale, void *stream);

/*
 * vdx_attn_fwd without any device allocation (the paper has no counterpart;
 * this is a library service).  Same arguments, results and errors as
 * vdx_attn_fwd -- the outputs are bit for bit those of vdx_attn_fwd, which
 * runs the same kernel with the same split -- for callers that cannot call
 * cudaMalloc during the call: code that runs while a stream is being
 * captured into a graph (an allocation there breaks the capture), a serving
 * loop whose device memory is planned before it starts, a process whose
 * device memory belongs to another allocator.
 *
 * Instead of the library's per-stream scratch, the split-tail scratch lives
 * in a fixed 24 MiB array of device memory inside the library image, which
 * every GPU that loads the library holds until the process exits.  A call
 * whose scratch need exceeds 24 MiB returns VDX_ERR_UNSUPPORTED and launches
 * nothing (with at most one part per multiprocessor the need stays near
 * 21 MB at D = 128 on a 152-SM GB300).
 *
 * Arguments are checked exactly as vdx_attn_fwd checks them, before any CUDA
 * call.  The first call on a device then looks up that array's device
 * address (once per device, the device being current); make that first call
 * before any stream capture.  Every call on a device shares the one array and
 * it keeps the previous call's contents: each call clears its counters
 * itself, on its stream, before the kernel.  Calls whose work overlaps on the
 * GPU (different streams, or threads without ordering) race on the array, so
 * order them.  No cudaMalloc, cudaFree or allocating library routine is
 * called.
 */
int vdx_attn_fwd_noalloc(const void *q, const void *k, const void *v, void *out, float *lse,
                         int B, int H, int Sq, int Skv, int D, float scale, void *stream);

/*
 * Attention forward on HOST buffers (a library service around Sec. 2's
 * attention op; the paper has no counterpart): vdx_attn_fwd, or
 * vdx_attn_fwd_varlen when kv_lens != NULL, for callers whose tensors live in
 * host memory.  The library copies the inputs in, runs the kernel and copies
 * the results out, overlapping the three: the (b, h) rows are cut into
 * chunks, and chunk i's kernel runs while chunk i+1 is copied in and chunk
 * i-1 copied out.
 *   q, k, v, out, lse, kv_lens : HOST pointers, caller-owned, laid out as in
 *          vdx_attn_fwd(_varlen) (kv_lens: int32 [B], read by the host during
 *          the call and copied in); lse may be NULL.  No alignment rule.  out
 *          and lse must not overlap each other or the inputs.
 *   chunk_rows : (b, h) rows per chunk; 0 lets the library choose from a
 *          cost model of the copies and the kernel.  With kv_lens, a chunk
 *          holds heads of one sample or whole samples (rounded down to a
 *          multiple of H above H).
 * Ordered after earlier work on `stream`, and `stream` waits for the last
 * copy out, so out and lse are complete once `stream` is synchronised; the
 * call itself returns once everything is enqueued.  Copies overlap only when
 * the host buffers are pinned (page-locked); pageable buffers give the same
 * results with the copies serialised by the CUDA runtime.  The host buffers
 * must stay valid until `stream` is synchronised.
 * Streams: besides `stream`, the library's own copy-in and copy-out streams
 * and two compute streams that alternate over the chunks (so that a chunk's
 * kernel fills the multiprocessors the previous one's last round leaves
 * idle).  Each chunk's kernel is vdx_attn_fwd(_varlen) on those rows, so the
 * results are bit for bit those of such calls.
 * Memory: per (device, stream), three device slots of one chunk's q, k, v,
 * out and lse each (~100 MB for B=1, H=12, S=32760, D=128 at the default
 * chunking of one row), allocated by the first call, grown by a larger one
 * (which waits for the device), kept until the process exits; plus
 * vdx_attn_fwd's workspace per compute stream.  Errors: as vdx_attn_fwd;
 * chunk_rows < 0 is VDX_ERR_INVALID_ARG.
 */
int vdx_attn_fwd_host(const void *q, const void *k, const void *v, void *out, float *lse,
                      int B, int H, int Sq, int Skv, int D, const int *kv_lens, float scale,
                      long long chunk_rows, void *stream);

/*
 * vdx_attn_fwd_rope3d on HOST buffers, through the same pipeline as
 * vdx_attn_fwd_host: each chunk's q and k rows are turned in place in the
 * device slot (the rotation works row by row, so a chunk turns exactly as
 * the whole tensor would) before the chunk's attention.  Arguments as
 * vdx_attn_fwd_rope3d plus chunk_rows; results: each chunk is vdx_rope3d on
 * its q and k rows followed by vdx_attn_fwd on those rows.  Errors as
 * vdx_attn_fwd_rope3d and vdx_attn_fwd_host.
 */
int vdx_attn_fwd_rope3d_host(const void *q, const void *k, const void *v, void *out, float *lse,
                             int B, int H, int S, int D, int F, int Hp, int Wp, int s0,
                             int d_t, int d_h, int d_w, float theta, int interleaved,
                             float scale, long long chunk_rows, void *stream);

/*
 * vdx_attn_fwd_segments on HOST buffers, through the same pipeline as
 * vdx_attn_fwd_host.  q_seg [B, Sq] and kv_seg [B, Skv] are HOST int32
 * arrays, copied in once per call; chunks hold heads of one sample or whole
 * samples.  Results and errors as vdx_attn_fwd_segments; memory as
 * vdx_attn_fwd_host plus B*(Sq+Skv) ints for the ids.
 */
int vdx_attn_fwd_segments_host(const void *q, const void *k, const void *v, void *out, float *lse,
                               int B, int H, int Sq, int Skv, int D, const int *q_seg, const int *kv_seg,
                               float scale, long long chunk_rows, void *stream);

/*
 * vdx_attn_fwd_win3d on HOST buffers, through the same pipeline as
 * vdx_attn_fwd_host (every (b, h) shares the grid, so a chunk is any block of
 * rows).  Results and errors as vdx_attn_fwd_win3d.
 */
int vdx_attn_fwd_win3d_host(const void *q, const void *k, const void *v, void *out, float *lse,
                            int B, int H, int F, int Hp, int Wp, int D, int kt, int kh, int kw,
                            int neighbourhood, float scale, long long chunk_rows, void *stream);

/*
 * Releases the device memory the library keeps for `stream` on the current
 * device (a library service; the paper has no counterpart): the split-tail
 * scratch and key-tile lists of the device calls, the turned q and k of
 * vdx_attn_fwd_rope3d, and the host-buffer pipeline (its device slots,
 * events and internal streams, and the scratch of its compute streams).
 * Synchronises `stream` and the pipeline's streams first.  The next call on
 * `stream` allocates again.  Call it only while no other thread enqueues work
 * on `stream` through this library.  Returns VDX_OK (also when nothing was
 * kept) or VDX_ERR_CUDA.
 */
int vdx_release(void *stream);

/* Human-readable name of a vdx_status (static storage; never NULL). */
const char *vdx_status_string(int status);

/*
 * Synchronises `stream`, then takes the library's device error word on the
 * current device: reads and zeroes it in one atomic exchange, so a bit a
 * kernel sets meanwhile is reported by this check or the next, never lost.
 * The word is per device, shared by every stream: a kernel on another stream
 * that gave up since the last check is reported here too.  Returns VDX_OK;
 * VDX_ERR_TIMEOUT if a kernel gave up on a bounded wait (its work stopped
 * cleanly: every copy and tensor-core operation it issued had finished before
 * it exited); VDX_ERR_DRAIN if a kernel could not confirm that (the GPU broke
 * a completion guarantee; treat device memory as suspect); VDX_ERR_CUDA if
 * the synchronisation or the read failed.  Checks from several threads are
 * serialised.
 */
int vdx_check_device_error(void *stream);

/*
 * Failure-detection self-test: launches one block whose only wait is on an
 * mbarrier that nothing ever arrives on, bounded by `limit_us` microseconds
 * (1 .. 10,000,000).  The kernel records VDX_ERR_TIMEOUT in the device error
 * word and returns; the GPU context stays usable.  Read the result with
 * vdx_check_device_error.  No fault, trap or hang is involved.
 */
int vdx_selftest_wait_timeout(int limit_us, void *stream);

/* Library version as major*10000 + minor*100 + patch. */
int vdx_version(void);

#ifdef __cplusplus
}
#endif

#endif /* VDX_H */
