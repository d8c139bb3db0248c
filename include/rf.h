/*
 * rf.h -- C ABI of the RhymeFlow asynchronous denoising step core on GB300.
 *
 * RhymeFlow (Sec. 3.2, Algorithm 2) denoises video latent frames on different
 * schedules: keyframes take one flow-matching step every timestep, non-keyframes
 * jump n_skip steps at once on their scheduled steps.  At every timestep only
 * the active frames issue attention queries; they attend to keys and values of
 * the whole latent sequence, in which the skipped frames are represented by a
 * linear projection of their latent trajectory (Eq. 3).  Afterwards only the
 * active frames take their Euler step.
 *
 * One step of that core is five calls, all asynchronous on a caller-provided
 * CUDA stream and all working on caller-owned device buffers:
 *
 *   rf_schedule_compact  active-frame mask -> frame / token index lists
 *   rf_project           Eq. 3 for skipped frames' latents, copy for active frames
 *   rf_project_kv        Eq. 3 for skipped frames' keys and values from the
 *                        rolling cache of Appendix B.2; fresh rows shifted in
 *   rf_attn              active-query x full-sequence attention (bf16, tcgen05)
 *   rf_step              Euler update of the active frames
 *
 * plus the host planner rf_plan_build that turns a keyframe set and a stride
 * schedule into the per-step masks and weights.
 *
 * Conventions common to every call:
 *  - Pointers named d_* are device pointers, h_* host pointers.  The caller owns
 *    every buffer; no call allocates, frees or retains memory beyond its return
 *    (rf_attn keeps a small per-process cache of device properties only), except
 *    the host-fed pipeline object, which owns its device memory from
 *    rf_pipeline_create to rf_pipeline_destroy.
 *  - `stream` is a cudaStream_t (NULL = the legacy default stream).  Work is
 *    enqueued and the call returns; nothing synchronises the host.
 *  - Errors that the host can see (null pointers, bad sizes, unsupported head
 *    dim, misalignment) are returned before anything is enqueued.  A failed
 *    kernel launch returns RF_ERR_CUDA.  Errors found on the device are written
 *    to the optional device status word of rf_attn and never trap or hang.
 *  - Frame-major latent layout: a latent state is [F][E] fp32 with E elements
 *    per frame (E = N*C for N tokens of C channels).  The two-slot store is
 *    [2][F][E]: slot cur_slot[f] holds frame f's current state and slot
 *    1-cur_slot[f] the state before its last jump (the "before"/"after" pair of
 *    Appendix B.2; shift-and-store is a slot flip, not a copy).
 */
#ifndef RF_H_
#define RF_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

struct CUstream_st;
typedef struct CUstream_st* rf_stream_t; /* == cudaStream_t */

typedef enum {
  RF_OK = 0,
  RF_ERR_INVALID_ARG = 1,     /* null pointer, negative or overflowing size */
  RF_ERR_UNSUPPORTED = 2,     /* e.g. head dim not in {64, 128}, no sm_103 device */
  RF_ERR_MISALIGNED = 3,      /* pointer or stride breaks a 16-byte TMA rule */
  RF_ERR_CUDA = 4,            /* a CUDA runtime call or kernel launch failed */
  RF_ERR_DEVICE_TIMEOUT = 5   /* a bounded device-side wait expired (status word) */
} rf_status;

/* Human-readable name of a status code.  Never NULL; static storage. */
const char* rf_status_str(int status);

/* Library ABI version (major*100 + minor). */
int rf_version(void);

/* Detail of the most recent non-OK status returned to the calling thread (which check
 * or CUDA call failed, with the CUDA error string), or "" if none.  Thread-local static
 * storage, valid until the thread's next call into the library. */
const char* rf_last_error(void);

/*
 * rf_plan_build -- host planner (CPU, deterministic): Algorithm 2 and Eq. 2.
 *
 * Steps s = 0..S-1 run from sigma_0 down to sigma_S = 0 (Algorithm 2's t = T..1).
 * A frame is active at step s if it is a keyframe, if s < T_w (synchronous
 * warm-up, Sec. 3.2.1), or if its state has reached step s (its "due" step).
 * An active keyframe (or any frame in warm-up) advances one step; an active
 * non-keyframe jumps h_stride[s] steps, the last jump clamped to sigma_S.
 * Under a constant stride this equals Algorithm 2's modulo rule.
 *
 *   F, S        frames, steps (F >= 1, S >= 1, F*S <= 2^31-1)
 *   h_is_key    [F]   nonzero = keyframe
 *   h_stride    [S]   skip stride per step, each >= 1
 *   T_w         warm-up steps, 0 <= T_w <= S
 *   h_sigma     [S+1] noise levels, strictly decreasing, sigma[S] = 0;
 *               NULL = uniform sigma_s = 1 - s/S
 * Outputs (caller-allocated host arrays, all [S][F] row-major):
 *   h_mask      1 = active at step s
 *   h_alpha     Eq. 3 weight for skipped frames,
 *               (sigma_start - sigma_s)/(sigma_start - sigma_due) computed in
 *               double and rounded to float; 1 for active frames; 0 when
 *               sigma_start == sigma_due
 *   h_beta      1 - alpha, computed in double and rounded to float
 *   h_dt        Euler step sigma_due - sigma_s for active frames, 0 otherwise
 *   h_cur_slot  slot of the two-slot store holding the frame's current state
 *               when step s begins (may be NULL)
 * Returns RF_ERR_INVALID_ARG on bad sizes / null pointers / stride < 1 / bad sigma.
 */
rf_status rf_plan_build(int F, int S, const uint8_t* h_is_key, const int32_t* h_stride, int T_w,
                        const double* h_sigma, uint8_t* h_mask, float* h_alpha, float* h_beta,
                        float* h_dt, uint8_t* h_cur_slot);

/*
 * rf_schedule_compact -- Algorithm 2's active set I_active as index lists.
 *
 *   d_mask       [F] uint8, nonzero = active
 *   F, N         frames (1..4096), tokens per frame (>= 1, F*N <= 2^31-1)
 * Outputs (device, caller-allocated):
 *   d_active     [F] int32: active frames ascending in [0, A); rest untouched
 *   d_skipped    [F] int32: skipped frames ascending in [0, F-A); rest untouched
 *   d_token_idx  [F*N] int32: f*N + p for each active f (ascending) and p < N,
 *                in [0, A*N); rest untouched.  May be NULL (not written).
 *   d_counts     [2] int32: {A, A*N}
 * Bit-exact; one launch.
 */
rf_status rf_schedule_compact(const uint8_t* d_mask, int F, int N, int32_t* d_active,
                              int32_t* d_skipped, int32_t* d_token_idx, int32_t* d_counts,
                              rf_stream_t stream);

/*
 * rf_project -- Eq. 3, latent trajectory projection, for every frame.
 *
 *   d_ctx       [F][E] fp32 output: the full-sequence context at sigma_s
 *   d_z2        [2][F][E] fp32 two-slot store (see conventions)
 *   d_cur_slot  [F] uint8, 0 or 1
 *   d_alpha, d_beta  [F] fp32 weights of this step (rf_plan_build row s)
 *   F, E        frames, elements per frame (E % 4 == 0; 16-byte aligned buffers)
 * For frame f with cur = z2[cur_slot[f]][f], prev = z2[1-cur_slot[f]][f]:
 *   beta[f] == 0:  ctx[f] = cur             (active frame: copy, prev not read)
 *   otherwise:     ctx[f] = fmaf(alpha[f], cur, beta[f]*prev)
 * d_ctx must not overlap d_z2.
 */
rf_status rf_project(float* d_ctx, const float* d_z2, const uint8_t* d_cur_slot,
                     const float* d_alpha, const float* d_beta, int F, int64_t E,
                     rf_stream_t stream);

/*
 * rf_project_kv -- per-layer rolling key/value cache (Appendix B.2), one layer, one
 * step, keys and values together.
 *
 *   d_K, d_V     bf16 attention inputs, row t = token at base + t*kv_row_stride,
 *                D contiguous elements (D = H*d, heads interleaved)
 *   d_Kc, d_Vc   bf16 two-slot caches [2][F][N][D] (slot cur_slot[f] = the frame's latest
 *                cached state "after", the other slot the state before it)
 *   d_cur_slot, d_alpha, d_beta  [F] this step's slot bits and Eq. 3 weights (the plan)
 *   d_active, d_skipped, d_counts  lists from rf_schedule_compact (device)
 *   F, N, D      frames, tokens per frame, elements per token (D % 8 == 0,
 *                kv_row_stride % 8 == 0, all bases 16-byte aligned)
 * For each skipped frame f its K and V rows are overwritten with
 *   bf16(fmaf(alpha[f], after, beta[f] * before))        (fp32 arithmetic, RNE)
 * and for each active frame its fresh K and V rows are copied into the cache's other
 * slot (the plan's slot flip then makes them "after": shift-and-store).  Rows of
 * active frames and caches of skipped frames are not written.  One launch.
 */
rf_status rf_project_kv(void* d_K, void* d_V, int64_t kv_row_stride, void* d_Kc, void* d_Vc,
                        const uint8_t* d_cur_slot, const float* d_alpha, const float* d_beta,
                        const int32_t* d_active, const int32_t* d_skipped,
                        const int32_t* d_counts, int F, int N, int D, rf_stream_t stream);

/*
 * rf_attn -- active-query x full-sequence softmax attention (Sec. 3.2.4 and
 * Appendix B.2: the active frames' queries attend to the keys and values of
 * all F*N tokens, true for active frames and projected for skipped ones).
 *
 *   d_O          bf16 output, row t at d_O + t*o_row_stride + h*d (t = token);
 *                only rows of active frames are written
 *   d_lse        fp32 [H][F*N] natural-log sum-exp per row, or NULL
 *   d_Q,d_K,d_V  bf16 inputs, row t head h at base + t*qkv_row_stride + h*d
 *   qkv_row_stride, o_row_stride  elements between tokens (>= H*d, % 8 == 0)
 *   F, N, H, d   frames, tokens/frame, heads, head dim (d in {64, 128})
 *   d_active     [F] int32 active frame list, d_counts [2] {A, ...}
 *                (as written by rf_schedule_compact; read on the device, so no
 *                host synchronisation is needed between the two calls)
 *   softmax_scale  scale applied to q.k (e.g. 1/sqrt(d))
 *   d_status     int32 device word or NULL: set nonzero if a bounded wait in
 *                the kernel expired (RF_ERR_DEVICE_TIMEOUT in bits 0..7); the
 *                caller clears it and reads it after synchronising
 * For each active frame f, token p < N, head h:
 *   O[f*N+p, h] = sum_j softmax_j(scale * q.k_j) v_j over all F*N tokens j.
 * Arithmetic: bf16 products, fp32 accumulation and softmax, probabilities
 * rounded to bf16 for the PV product, output rounded to bf16.
 *   d_workspace, workspace_bytes  optional device scratch for split-KV (NULL / 0 =
 *                no split).  With at least rf_attn_workspace_bytes(d) bytes, 256-byte
 *                aligned and ZERO-FILLED before its first use, the last, partly
 *                idle round of work is split into ranges of keys whose partial
 *                results are merged on the device; the kernel leaves the workspace
 *                ready for the next call.  Calls that share a workspace must not
 *                overlap on the GPU (keep them on one stream).  After a call that
 *                reported RF_ERR_DEVICE_TIMEOUT, zero it again.
 * Requires an sm_103 device; bases 16-byte aligned.
 */
rf_status rf_attn(void* d_O, float* d_lse, const void* d_Q, const void* d_K, const void* d_V,
                  int64_t qkv_row_stride, int64_t o_row_stride, int F, int N, int H, int d,
                  const int32_t* d_active, const int32_t* d_counts, float softmax_scale,
                  void* d_workspace, int64_t workspace_bytes, int32_t* d_status,
                  rf_stream_t stream);

/*
 * rf_attn_block_masked -- rf_attn under the combined mask of Appendix D:
 * M_combined = M_Rhyme (element-wise) M_SAP.  M_Rhyme, the frame mask, is the active list
 * (only active frames' queries are computed, as in rf_attn); M_SAP is a token-level block
 * mask:
 *   d_block_mask  uint8 [H][nb][nb], nb = ceil(F*N / 128): entry [h][qb][kb] nonzero lets
 *                 query tokens 128*qb .. 128*qb+127 attend to key tokens 128*kb .. 128*kb+127
 *                 for head h (blocks over the token index t = f*N + p of the whole sequence)
 * Keys a row may not attend to are excluded from its softmax; key blocks no query row of a
 * work item may attend to are not loaded or multiplied at all.  A row that may attend to
 * no key gets O = 0 and LSE = -inf.  All other arguments, requirements and results are
 * those of rf_attn, except for the workspace: the work is never split into KV ranges, and
 * with a workspace (same size and rules as for rf_attn) a small pre-pass launch orders the
 * work items longest first within groups of heads and the CTAs take them from a queue.  The
 * queue and the groups use the workspace's counter words, which the calls leave at zero, and
 * the items' costs and order use its partial-row area.  Without a workspace, items are dealt
 * round-robin.  Returns RF_ERR_INVALID_ARG for a null mask and RF_ERR_UNSUPPORTED for more
 * than 4096 key blocks (F*N > 524288 tokens).
 */
rf_status rf_attn_block_masked(void* d_O, float* d_lse, const void* d_Q, const void* d_K,
                               const void* d_V, int64_t qkv_row_stride, int64_t o_row_stride,
                               int F, int N, int H, int d, const int32_t* d_active,
                               const int32_t* d_counts, float softmax_scale,
                               const uint8_t* d_block_mask, void* d_workspace,
                               int64_t workspace_bytes, int32_t* d_status, rf_stream_t stream);

/*
 * rf_attn_workspace_bytes -- bytes of split-KV workspace rf_attn can use on the
 * current device for head dim d (independent of the problem size: counters plus
 * one partial result tile per SM).  Returns -1 for an unsupported d or when the
 * device cannot be queried.
 */
int64_t rf_attn_workspace_bytes(int d);

/*
 * rf_attn_noalloc -- rf_attn for callers that cannot allocate device memory.
 *
 * The paper has no counterpart to this entry point; it exists for deployment.
 * Some callers of this library cannot call cudaMalloc: code running inside
 * another engine's execution callback that forbids allocation, serving loops
 * that must not take cudaMalloc's implicit device-wide synchronisation, or plain
 * C hosts with no device allocator of their own.  For them this call takes the
 * same arguments as rf_attn minus the workspace, and uses instead a scratch
 * array that the library itself holds in device memory: a file-scope array of
 * 21,630,976 bytes (split-KV counters plus partial tiles for head dim <= 128 on
 * up to 160 SMs), present on every GPU that loads the library until the
 * process exits.  The call allocates and frees nothing.
 *   - The first call on a device looks up the array's device address
 *     (cudaGetSymbolAddress) with that device current and caches it for the
 *     life of the process; make that first call before any stream capture.
 *     cudaDeviceReset (or any other teardown of the device's primary context)
 *     invalidates the cached address: do not call rf_attn_noalloc on a device
 *     after resetting it.
 *   - Argument errors (those rf_attn returns) are returned before anything is
 *     enqueued.  Otherwise each call zeroes the array's counters on `stream`
 *     before the kernel runs.
 *   - Every call on a device shares the one array, and it keeps the last call's
 *     contents: calls that overlap on the GPU (different streams, or several
 *     host threads) race on it and give wrong results.  Issue them in order on
 *     one stream.
 *   - If the device needs more scratch than the array holds (more than 160
 *     SMs), the call returns RF_ERR_UNSUPPORTED with the sizes in
 *     rf_last_error(); nothing is enqueued.
 * The inputs, outputs and results are those of rf_attn with a workspace.
 */
rf_status rf_attn_noalloc(void* d_O, float* d_lse, const void* d_Q, const void* d_K,
                          const void* d_V, int64_t qkv_row_stride, int64_t o_row_stride, int F,
                          int N, int H, int d, const int32_t* d_active, const int32_t* d_counts,
                          float softmax_scale, int32_t* d_status, rf_stream_t stream);

/*
 * rf_step -- heterogeneous flow-matching Euler update (Sec. 3.2.3, Algorithm 2):
 * each active frame f takes z_next = z + dt[f] * v (dt = sigma_due - sigma_s;
 * one step for keyframes, n_skip steps for non-keyframes).
 *
 *   d_z2        [2][F][E] fp32 two-slot store: reads slot cur_slot[f], writes
 *               slot 1-cur_slot[f] with fmaf(dt[f], v, z); the caller then flips
 *               cur_slot[f] for the active frames (rf_plan_build does this)
 *   d_cur_slot  [F] uint8
 *   d_v         [F][E] fp32 velocity
 *   d_dt        [F] fp32
 *   d_active, d_counts  active list from rf_schedule_compact (device)
 *   F, E        frames, elements per frame (E % 4 == 0; 16-byte aligned)
 */
rf_status rf_step(float* d_z2, const uint8_t* d_cur_slot, const float* d_v, const float* d_dt,
                  const int32_t* d_active, const int32_t* d_counts, int F, int64_t E,
                  rf_stream_t stream);

/*
 * rf_frame_gram -- inner products of the F clean-latent proxies, the input of sequential
 * keyframe selection (Sec. 3.1, Eq. 1; Algorithm 1 compares frames by cosine similarity).
 *
 *   d_P   fp32 [F][ld] proxies (frame f's E elements at d_P + f*ld), 1 <= F <= 64, ld >= E
 *   d_G   fp64 [F][F] output, G[i][j] = sum_e P[i][e] * P[j][e]; the call zero-fills it on
 *         `stream` first (partial sums are added with atomics, so summation order varies
 *         between runs at the level of fp64 rounding)
 * Per-CTA partial products are fp32 (each over at most E / #SMs / 2 elements), accumulated
 * across CTAs in fp64.
 */
rf_status rf_frame_gram(const float* d_P, int F, int64_t E, int64_t ld, double* d_G,
                        rf_stream_t stream);

/*
 * rf_keyframe_select -- Algorithm 1 (dynamic sequential keyframe selection) on the host,
 * over a host copy of rf_frame_gram's result.
 *
 *   h_G        fp64 [F][F] inner products (diagonal > 0)
 *   M          keyframe budget (>= 1); tau, dtau, delta_up, delta_down as in Algorithm 1
 *              (the paper gives no values)
 *   h_is_key   [F] output, 1 = keyframe; h_num_keys (nullable) output count
 * Frame 0 is always a keyframe.  Visiting frames in order while fewer than M keyframes
 * exist, a frame whose cosine similarity to the latest keyframe is below tau becomes one;
 * first tau -= dtau if the gap to the latest keyframe is >= F/M + delta_up, or
 * tau += dtau if it is <= F/M - delta_down (Algorithm 1 as printed; a negative dtau gives
 * the adjustment direction its prose describes).
 */
rf_status rf_keyframe_select(const double* h_G, int F, int M, double tau, double dtau,
                             double delta_up, double delta_down, uint8_t* h_is_key,
                             int32_t* h_num_keys);

/*
 * rf_pipeline -- the step core fed from pinned host memory: one asynchronous denoising step
 * (Algorithm 2: rf_schedule_compact, rf_project, rf_project_kv, rf_attn, rf_step) per
 * rf_pipeline_step, with the step's inputs copied from the host and its results copied back,
 * the copies of neighbouring steps overlapped with the compute of the current one.  The keys
 * and values of skipped frames never cross the bus: they are the Eq. 3 projection of the
 * device-resident rolling cache (Appendix B.2).  No paper passage: this is the host side of
 * serving the step core.
 *
 * rf_pipeline_create allocates, on the current device, the plan, the two-slot latent store,
 * the rolling key/value cache (bf16 [2][F][N][H*d] each), the index lists, an rf_attn
 * workspace and `depth` buffer sets (Q, K, V, O bf16 [F*N][H][d]; velocity fp32 [F][E];
 * snapshots of the latent store fp32 [2][F][E] and of the context fp32 [F][E]).
 *   h_mask, h_alpha, h_beta, h_dt, h_cur_slot  the plan, [S][F] as rf_plan_build writes it
 *   h_z2        fp32 [2][F][E] initial two-slot latent store
 *   h_K0, h_V0  bf16 [F*N][H][d] initial keys and values: both cache slots of every frame
 *               start with them (the cache's counterpart of both latent slots holding z0)
 *   depth       buffer sets, 2..8 (3 lets a heavy step's input copies run during the two
 *               steps before it)
 *   compute, h2d, d2h  three streams the pipeline enqueues on (all work of a step is
 *               ordered by events recorded on them; the caller may record its own events)
 *   *out        the pipeline; RF_ERR_* and *out = NULL on failure (nothing leaks)
 * d in {64, 128}; E % 4 == 0.
 *
 * rf_pipeline_step enqueues schedule step s (0 <= s < S) and returns:
 *   h_Q, h_K, h_V  pinned host bf16 [F*N][H][d] (rows contiguous): the fresh queries, keys
 *               and values; only the rows of the frames active at step s are read
 *   h_v         pinned host fp32 [F][E] velocity of the step
 *   h_O         pinned host bf16 [F*N][H][d]: the active frames' rows are written
 *   h_z2        pinned host fp32 [2][F][E]: the latent store after the step
 *   h_ctx       pinned host fp32 [F][E] (nullable): the step's Eq. 3 latent context
 *   softmax_scale  as for rf_attn
 * Host buffers of a step must stay valid and untouched until rf_pipeline_sync; the buffers
 * of `depth` consecutive steps may be in flight at once.  A step that returns an error may
 * have enqueued part of its work, and the order between later steps is then not kept: after
 * an error, call rf_pipeline_sync (to drain) and rf_pipeline_destroy.
 *
 * rf_pipeline_sync waits for every enqueued step and writes the device status word (as for
 * rf_attn) to *h_status (nullable).  rf_pipeline_bytes reports the steps enqueued and the
 * host->device and device->host bytes they copy.  rf_pipeline_destroy waits and frees
 * everything (NULL is ignored).
 */
typedef struct rf_pipeline rf_pipeline;
rf_status rf_pipeline_create(int F, int N, int H, int d, int64_t E, int S,
                             const uint8_t* h_mask, const float* h_alpha, const float* h_beta,
                             const float* h_dt, const uint8_t* h_cur_slot, const float* h_z2,
                             const void* h_K0, const void* h_V0, int depth,
                             rf_stream_t compute, rf_stream_t h2d, rf_stream_t d2h,
                             rf_pipeline** out);
rf_status rf_pipeline_step(rf_pipeline* p, int s, const void* h_Q, const void* h_K,
                           const void* h_V, const float* h_v, void* h_O, float* h_z2,
                           float* h_ctx, float softmax_scale);
rf_status rf_pipeline_sync(rf_pipeline* p, int32_t* h_status);
rf_status rf_pipeline_bytes(const rf_pipeline* p, int64_t* h_steps, int64_t* h_h2d_bytes,
                            int64_t* h_d2h_bytes);
void rf_pipeline_destroy(rf_pipeline* p);

/*
 * rf_selftest_bounded_wait -- check, on the GPU, the path every device-side wait
 * of rf_attn takes when it runs out of time.  No paper passage: this is a
 * failure-handling self-test.
 *
 * Launches one CTA that allocates tensor memory, waits on an mbarrier that
 * nothing ever arrives at, gives up after limit_us microseconds
 * (100 <= limit_us <= 2,000,000), ORs RF_ERR_DEVICE_TIMEOUT into *d_status,
 * frees its tensor memory and returns.  Nothing faults or traps and the context
 * stays usable.  The caller zeroes *d_status first and reads it after
 * synchronising.  Returns RF_ERR_INVALID_ARG for a null pointer or an out-of-range
 * limit.
 */
rf_status rf_selftest_bounded_wait(int32_t* d_status, int limit_us, rf_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* RF_H_ */
