/*
 * fsx.h -- C ABI of the GB300 action-expert tick.
 *
 * The fast system of an asynchronous fast-slow driving agent ("Think at 5 Hz,
 * Act at 20 Hz", Sec. 3.1 and Sec. 3.3): a 32-layer action expert whose tokens,
 * at every layer l, attend over the concatenation of the frozen backbone's
 * layer-l KV cache and the expert's own keys/values (Eq. 1), followed by an
 * output projection, a SwiGLU block and a waypoint head. One call = one tick.
 *
 * Conventions for every entry point:
 *   - Pointers marked "device" must point to memory of the handle's device;
 *     "host" pointers to ordinary (pageable or pinned) host memory.
 *   - The caller owns every buffer it passes; the library never frees,
 *     retains or writes any caller buffer except the documented outputs.
 *   - Streams are passed as void* holding a cudaStream_t (NULL = legacy
 *     default stream). Work is enqueued asynchronously unless stated.
 *   - Every function returns an fsx_status; on failure a thread-local message
 *     is available from fsx_last_error(). Host-side argument checks happen
 *     before anything is enqueued.
 *   - Supported shapes: head_dim == 128, d_model % 128 == 0, d_model <= 1024,
 *     d_ff % 64 == 0, 1 <= n_action + n_frame <= 48, 1 <= n_waypoints <=
 *     n_action + n_frame, n_layers <= 128. Other shapes give FSX_ERR_UNSUPPORTED.
 *   - Precision: weights are stored as fp16 (round-to-nearest-even from the
 *     fp32 host copy; exact for bf16-valued weights), GEMM and attention
 *     operands are fp16 with fp32 accumulation, the residual stream, RMSNorm,
 *     softmax statistics and the head are fp32. Cache values the kernels
 *     convert to fp16 (every key; the values too, except in the bf16 tensor-core
 *     attention of batched ticks, which keeps them bf16) must lie within
 *     +-65504. A value beyond that (a bf16 magnitude of 65536 or more, an fp32
 *     magnitude that rounds past 65504, infinity or NaN) is a device-side error:
 *     the status becomes FSX_ERR_RANGE and the tick is abandoned like on bad
 *     offsets, writing no waypoint, instead of returning NaN waypoints. In the
 *     tensor-core attention the check is made on the scores: a key beyond the
 *     range whose scores all fall to -inf has weight zero, as its exact value
 *     would, and is not reported.
 */
#ifndef FSX_H
#define FSX_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct fsx_handle_s* fsx_handle;

typedef enum {
  FSX_OK = 0,
  FSX_ERR_INVALID_ARG = 1,  /* a host-checked argument is wrong                */
  FSX_ERR_UNSUPPORTED = 2,  /* a shape or dtype outside the supported set      */
  FSX_ERR_OOM = 3,          /* a device or host allocation failed              */
  FSX_ERR_CUDA = 4,         /* a CUDA runtime call failed (see fsx_last_error) */
  FSX_ERR_TIMEOUT = 5,      /* a bounded device-side wait gave up              */
  FSX_ERR_DEVICE_ARG = 6,   /* device-side check: offsets not non-decreasing,
                               negative, or beyond max_total_cache_tokens      */
  FSX_ERR_RANGE = 7         /* device-side check: a cache value lies outside
                               the fp16 range (see Precision)                  */
} fsx_status;

typedef enum { FSX_F32 = 0, FSX_BF16 = 1 } fsx_dtype;

/* Model and capacity description, fixed at fsx_create. */
typedef struct {
  int n_layers;      /* expert layers == backbone layers (32); layer l reads cache layer l */
  int d_model;       /* expert width d_ae (512)                                     */
  int n_heads;       /* backbone attention heads (32)                               */
  int head_dim;      /* backbone head width (128)                                   */
  int d_ff;          /* SwiGLU hidden width (1408)                                  */
  int n_action;      /* learned action tokens per vehicle (10)                      */
  int n_frame;       /* frame tokens per vehicle (32)                               */
  int n_waypoints;   /* waypoints per vehicle, read from action tokens 0.. (5)      */
  int max_batch;     /* largest B any later fsx_tick may pass                       */
  long long max_total_cache_tokens; /* largest offsets[B] any later tick may pass   */
  int cache_dtype;   /* fsx_dtype of the K/V cache rows                             */
  int frame_dtype;   /* fsx_dtype of the frame tokens                               */
} fsx_config;

/* Host fp32 expert weights, copied (and converted) by fsx_create; every matrix
 * is row-major [out_features, in_features] and stacked over layers. */
typedef struct {
  const float* act_emb;    /* [n_action, d]                     learned action tokens  */
  const float* pos_emb;    /* [n_action + n_frame, d]           learned positions      */
  const float* attn_norm;  /* [n_layers, d]                     RMSNorm gain, attention*/
  const float* wq;         /* [n_layers, n_heads*head_dim, d]   W_q (Sec. 3.1)         */
  const float* wk;         /* [n_layers, n_heads*head_dim, d]   W_k                    */
  const float* wv;         /* [n_layers, n_heads*head_dim, d]   W_v                    */
  const float* wo;         /* [n_layers, d, n_heads*head_dim]   output projection      */
  const float* mlp_norm;   /* [n_layers, d]                     RMSNorm gain, SwiGLU   */
  const float* w_gate;     /* [n_layers, d_ff, d]               SwiGLU gate            */
  const float* w_up;       /* [n_layers, d_ff, d]               SwiGLU up              */
  const float* w_down;     /* [n_layers, d, d_ff]               SwiGLU down            */
  const float* final_norm; /* [d]                               RMSNorm gain, head     */
  const float* head_w;     /* [2, d]                            waypoint head          */
  const float* head_b;     /* [2]                               waypoint head bias     */
} fsx_weights;

/* Create a handle on `device`: validates cfg (host), uploads fp16 weights in
 * the kernels' tile order, allocates workspace for cfg->max_batch vehicles.
 * Blocking. Errors: INVALID_ARG (null/negative fields), UNSUPPORTED (shape),
 * OOM, CUDA. Env FSX_TEST_FAIL_ALLOC=1 forces the OOM path (tests);
 * FSX_PAIR_GEMM=1 runs the batched QKV projection (2048 tokens or more) on CTA
 * pairs (tcgen05.mma.cta_group::2) instead of single CTAs, with the same
 * results to rounding; FSX_DISABLE_PERSISTENT=1 (read at every tick) runs a
 * single vehicle through the batched graph instead of the one-launch tick. */
fsx_status fsx_create(const fsx_config* cfg, const fsx_weights* w, int device, fsx_handle* out);

/* One expert tick for B vehicles (Sec. 3.1, Eq. 1; Sec. 3.3: the cache is read
 * as-is and never written).
 *   k_cache, v_cache : HOST arrays of n_layers DEVICE pointers; layer l points
 *                      to [total_tokens, n_heads, head_dim] rows of
 *                      cfg.cache_dtype, token-major, vehicle b owning rows
 *                      offsets[b] .. offsets[b+1]-1. Read only. A layer
 *                      pointer may be NULL only when every L_b is 0.
 *   d_offsets        : DEVICE int64 [B+1], non-decreasing, offsets[0] >= 0,
 *                      offsets[B] <= max_total_cache_tokens. L_b may be 0.
 *   B                : 1 .. max_batch.
 *   d_frames         : DEVICE [B, n_frame, d_model] of cfg.frame_dtype.
 *   d_waypoints      : DEVICE fp32 [B, n_waypoints, 2] output.
 * Enqueued on `stream` as one CUDA-graph launch (plus a small argument upload
 * when any pointer changed since the previous tick); no host synchronisation.
 * Device-side checks (offsets) set a sticky status read by fsx_get_status;
 * the rest of that tick then reads no cache row and writes no waypoint. A handle must not run
 * two ticks concurrently; ticks on different streams are serialised by the
 * handle. Must not be called while `stream` is being captured. */
fsx_status fsx_tick(fsx_handle h, const void* const* k_cache, const void* const* v_cache,
                    const int64_t* d_offsets, int B, const void* d_frames,
                    float* d_waypoints, void* stream);

/* fsx_tick with an explicit first row per vehicle, for caches whose vehicles do not
 * lie back to back: vehicle b reads rows d_starts[b] .. d_starts[b] + L_b - 1 with
 * L_b = offsets[b+1] - offsets[b]. The ranges may leave gaps (room for the slow
 * system's appends) or overlap (prefixes of one shared cache, as in the
 * staleness-masked forward over a clip, Sec. 3.2). d_starts: DEVICE int64 [B], each
 * >= 0 with d_starts[b] + L_b <= max_total_cache_tokens (checked on the device);
 * d_offsets: DEVICE int64 [B+1], non-decreasing, giving only the lengths here (its
 * last entry may exceed max_total_cache_tokens). NULL d_starts is fsx_tick.
 * Everything else as fsx_tick. */
fsx_status fsx_tick_ranges(fsx_handle h, const void* const* k_cache, const void* const* v_cache,
                           const int64_t* d_starts, const int64_t* d_offsets, int B, const void* d_frames,
                           float* d_waypoints, void* stream);

/* fsx_tick with HOST frames, offsets and waypoints: copies h_offsets [B+1]
 * and h_frames [B, n_frame, d] to handle-owned device buffers, runs the
 * tick, copies the waypoints back to h_waypoints [B, n_waypoints, 2] and
 * synchronises `stream`. The caches stay device-resident (k/v as in fsx_tick). */
fsx_status fsx_tick_host(fsx_handle h, const void* const* k_cache, const void* const* v_cache,
                         const int64_t* h_offsets, int B, const void* h_frames,
                         float* h_waypoints, void* stream);

/* Same tick, launched kernel by kernel (no graph), additionally copying every
 * layer's Eq. 1 output (before W_o) to d_attn_out: DEVICE fp16
 * [n_layers, B*(n_action+n_frame), n_heads*head_dim]. For tests. */
fsx_status fsx_tick_debug(fsx_handle h, const void* const* k_cache, const void* const* v_cache,
                          const int64_t* d_offsets, int B, const void* d_frames,
                          float* d_waypoints, void* d_attn_out, void* stream);

/* fsx_tick_debug with the per-vehicle first rows of fsx_tick_ranges. For tests. */
fsx_status fsx_tick_ranges_debug(fsx_handle h, const void* const* k_cache, const void* const* v_cache,
                                 const int64_t* d_starts, const int64_t* d_offsets, int B, const void* d_frames,
                                 float* d_waypoints, void* d_attn_out, void* stream);

/* Status of the handle's ticks since the previous call. Not a passage of the
 * paper: the error path of the tick (Sec. 3.3 runs it every 50 ms, so a failed
 * tick must be detectable without stopping the stream). Synchronises `stream`
 * (the stream of the ticks to check), then returns and clears the device status
 * word: FSX_OK, FSX_ERR_DEVICE_ARG, FSX_ERR_TIMEOUT or FSX_ERR_RANGE (the first
 * error of those ticks; the tick that raised it wrote no waypoint). */
fsx_status fsx_get_status(fsx_handle h, void* stream);

/* For tests of the timeout path: the limit, in nanoseconds of the GPU's global timer,
 * of the single-launch tick's device-wide waits (B = 1), 1 s by default (limit_ns = 0
 * restores it). Not a passage of the paper. With a tiny limit a wait that finds its
 * counter incomplete gives up at once: the tick ends with FSX_ERR_TIMEOUT and writes no
 * waypoint, after letting everything it has in flight complete. Later ticks capture
 * their graphs again with the new limit. Must not be called while ticks run. */
fsx_status fsx_set_wait_limit(fsx_handle h, unsigned long long limit_ns);

/* Thread-local message describing the last failure on this thread ("" if none). */
const char* fsx_last_error(void);

/* Releases the handle's device memory and graphs (synchronises its device). */
void fsx_destroy(fsx_handle h);

/* Bytes of the handle's fp16 weight arena (algorithmic weight bytes per tick). */
long long fsx_weight_bytes(fsx_handle h);

/* Kernel launches one tick performs for batch B (what a graph replay runs). */
int fsx_tick_launches(fsx_handle h, int B);

/* Per-kernel-class timing of graph ticks, for roofline reports. With enable=1
 * later fsx_tick calls replay a graph variant that records CUDA events around
 * every launch of kernel class `kclass` (0 = QKV projection, 1 = attention,
 * 2 = output projection, 3 = SwiGLU gate/up, 4 = down projection, 5 = persistent
 * tick). fsx_kernel_time
 * returns the summed event time (ms) and launch count of the most recent tick
 * (synchronises the stream of that tick). Class 5 times the single-launch
 * persistent tick used for B = 1 (then fsx_tick_launches(h, 1) == 1). */
fsx_status fsx_set_kernel_timing(fsx_handle h, int enable, int kclass);
fsx_status fsx_kernel_time(fsx_handle h, float* ms, int* launches);

/* Eq. 1 alone (split-KV attention over [cache ; own], then the merge of the
 * splits), for B vehicles and every head, fp16 in / fp16 out.
 *   d_q      : DEVICE fp16, query row i of vehicle b at d_q + (b*n_q+i)*q_stride,
 *              n_heads*head_dim wide (head h at column h*head_dim).
 *   d_k_own, d_v_own : DEVICE fp16, own key/value row j of vehicle b at
 *              + (b*n_own+j)*own_stride (same column layout).
 *   d_k_cache, d_v_cache, d_offsets : as one layer of fsx_tick.
 *   n_q in 1..48, n_own >= 0, n_splits in 1..64 (keys of vehicle b are cut
 *   into n_splits near-equal ranges), head_dim == 128.
 *   d_out    : DEVICE fp16 [B*n_q, n_heads*head_dim].
 *   d_lse    : DEVICE fp32 [B, n_heads, n_q] natural-log log-sum-exp of the
 *              scaled scores, or NULL.
 *   d_workspace : DEVICE scratch of fsx_attention_workspace_bytes(...) bytes:
 *              a status word, then the per-split partial outputs. Only this
 *              call's kernels touch it; it must not be shared by calls that
 *              overlap on the GPU. Asynchronous on `stream`; cache offsets
 *              outside [0, ...] non-decreasing order make the kernels write
 *              nothing. */
size_t fsx_attention_workspace_bytes(int B, int n_heads, int n_q, int n_splits);
fsx_status fsx_attention(const void* d_q, long long q_stride,
                         const void* d_k_own, const void* d_v_own, long long own_stride,
                         int n_q, int n_own,
                         const void* d_k_cache, const void* d_v_cache, int cache_dtype,
                         const int64_t* d_offsets, int B, int n_heads, int head_dim,
                         int n_splits, void* d_out, float* d_lse,
                         void* d_workspace, size_t workspace_bytes, void* stream);

/* fsx_attention without any scratch argument and without any allocation.
 * The paper has no counterpart: this entry point exists for callers that may
 * not allocate device memory once they are running and cannot lend a scratch
 * buffer either -- e.g. a real-time vehicle stack that reserves all GPU memory
 * at start-up, because a run-time cudaMalloc can stall on a device-wide
 * synchronisation or fail under fragmentation, which a 50 ms control tick
 * cannot absorb. Arguments and results are those of fsx_attention. The
 * scratch is a 4 MiB array inside the library image, held on every GPU that
 * loads the library until the process exits; calls for which
 * fsx_attention_workspace_bytes(B, n_heads, n_q, n_splits) exceeds 4 MiB are
 * rejected with FSX_ERR_INVALID_ARG before anything is enqueued (n_splits = 1
 * needs only the status word, for any B). All calls on a device share
 * that array, so calls whose kernels overlap on the GPU race and must be
 * serialised by the caller. The first call on each device resolves the array's
 * device address with that device current; make it before capturing a stream.
 * The resolved address is kept for the process: it does not survive a reset of
 * the device's context (cudaDeviceReset), after which these entry points must
 * not be used. Unlike fsx_attention, whose status word sits in the caller's
 * workspace, device-side argument errors (cache offsets that are negative or
 * decrease: the vehicle concerned writes no output row) are recorded in the
 * static array; read them with fsx_attention_noalloc_status.
 * Allocates nothing: no cudaMalloc, cudaFree or allocating library call. */
fsx_status fsx_attention_noalloc(const void* d_q, long long q_stride,
                                 const void* d_k_own, const void* d_v_own, long long own_stride,
                                 int n_q, int n_own,
                                 const void* d_k_cache, const void* d_v_cache, int cache_dtype,
                                 const int64_t* d_offsets, int B, int n_heads, int head_dim,
                                 int n_splits, void* d_out, float* d_lse, void* stream);

/* The device status word of fsx_attention_noalloc's static array on the current
 * device (the paper has no counterpart; it completes that entry point for the
 * same callers). Synchronises `stream` -- the stream of the calls to check --
 * then returns the word and clears it: FSX_OK, FSX_ERR_DEVICE_ARG (a call saw
 * negative or decreasing cache offsets), FSX_ERR_TIMEOUT or FSX_ERR_RANGE (a
 * cache value outside the fp16 range, as in fsx_get_status). Copies one int to the
 * host and clears it on the device; allocates nothing. Calls still running on
 * other streams may set the word afterwards. */
fsx_status fsx_attention_noalloc_status(void* stream);

/* ============================================================ the paper's ten-token expert
 * Sec. 3.1 gives the expert ten tokens per vehicle and frame: one state token that
 * embeds the ego state -- the previous five predicted waypoints (x, y), the previous
 * control triplet (throttle, steer, brake), the current speed and the target point
 * (x, y), 16 values in that order -- the current frame's four visual tokens, and five
 * learned waypoint queries; a two-layer head decodes the five query outputs into five
 * (x, y) waypoints. The layer stack is the tick above.
 *   state token  t = W_s2 silu(W_s1 s + b_s1) + b_s2
 *   tokens       X = [t ; V (4 visual tokens) ; E_q (5 queries)] + P_pos
 *   waypoint i   w_i = W_h2 silu(W_h1 RMSNorm(X_{5+i}; g_f) + b_h1) + b_h2
 * Host fp32 weights, every matrix row-major [out_features, in_features], copied at
 * create; the layer weights are those of fsx_weights. */
typedef struct {
  const float* state_w1;   /* [d, 16]    state MLP, first layer    */
  const float* state_b1;   /* [d]                                  */
  const float* state_w2;   /* [d, d]     state MLP, second layer   */
  const float* state_b2;   /* [d]                                  */
  const float* query_emb;  /* [5, d]     learned waypoint queries   */
  const float* pos_emb;    /* [10, d]    positions: state, visual 0-3, queries 0-4 */
  const float* attn_norm;  /* [n_layers, d]   as fsx_weights       */
  const float* wq;         /* [n_layers, n_heads*head_dim, d]      */
  const float* wk;
  const float* wv;
  const float* wo;         /* [n_layers, d, n_heads*head_dim]      */
  const float* mlp_norm;   /* [n_layers, d]                        */
  const float* w_gate;     /* [n_layers, d_ff, d]                  */
  const float* w_up;
  const float* w_down;     /* [n_layers, d, d_ff]                  */
  const float* final_norm; /* [d]        RMSNorm gain before the head */
  const float* head_w1;    /* [d, d]     head, first layer          */
  const float* head_b1;    /* [d]                                   */
  const float* head_w2;    /* [2, d]     head, second layer         */
  const float* head_b2;    /* [2]                                   */
} fsx_paper_weights;

/* A tick handle for the ten-token layout (Sec. 3.1). cfg as for fsx_create, except
 * that n_action, n_frame and n_waypoints are fixed by the layout (5 queries, the
 * state token + 4 visual tokens, 5 waypoints; the given values are ignored) and
 * frame_dtype is the dtype of the visual tokens. The handle is an fsx_handle: use
 * fsx_paper_tick for its ticks, fsx_get_status, fsx_set_kernel_timing,
 * fsx_kernel_time and fsx_destroy as usual. Blocking. Errors as fsx_create. */
fsx_status fsx_paper_create(const fsx_config* cfg, const fsx_paper_weights* w, int device, fsx_handle* out);

/* One tick of the ten-token layout for B vehicles (Sec. 3.1, Eq. 1).
 *   k_cache, v_cache, d_offsets : as fsx_tick.
 *   d_visual    : DEVICE [B, 4, d] visual tokens of the current frame (cfg.frame_dtype).
 *   d_state     : DEVICE fp32 [B, 16] ego state (order above).
 *   d_waypoints : DEVICE fp32 [B, 5, 2] output.
 * Enqueued on `stream`: the state MLP writes the frame rows into a handle-owned
 * buffer, then the tick runs; device-side errors as fsx_tick (no waypoint written). */
fsx_status fsx_paper_tick(fsx_handle h, const void* const* k_cache, const void* const* v_cache,
                          const int64_t* d_offsets, int B, const void* d_visual, const float* d_state,
                          float* d_waypoints, void* stream);

/* ================================================================== cache append
 * The slow system's incremental forward (Sec. 1, Sec. 3.3): every K = 4 ticks
 * the current frame's n_new (4) tokens go through the frozen backbone -- a
 * causal, LLaMA-style decoder -- and every layer appends their keys (after the
 * rotary embedding) and values to its KV cache, the cache fsx_tick reads. The
 * cost does not depend on the history length, and rotary phases make the
 * append exact against a monolithic forward over the whole history.
 * Per layer, for the new token rows x of one vehicle:
 *   N = RMSNorm(x; g1, eps 1e-6);  q, k, v = N W_q^T, N W_k^T, N W_v^T;
 *   q, k rotated at their positions (dims j and j + head_dim/2 of a head turn
 *   by pos * rope_base^(-2j/head_dim); cached token i of a vehicle sits at
 *   position i, so the new tokens take positions L_b .. L_b + n_new - 1);
 *   causal attention over [the vehicle's cached rows ; the new rows];
 *   x += o W_o^T;  N = RMSNorm(x; g2);  x += (silu(N W_g^T) * (N W_u^T)) W_d^T.
 * Precision: weights fp16 (RNE from the fp32 host copy), GEMM operands fp16
 * with fp32 accumulation, fp32 residual stream, RMSNorm, rotation and softmax;
 * the cache rows are bf16 and the new rows are rounded to bf16 when written. */
typedef struct fsx_append_s* fsx_append_handle;

typedef struct {
  int n_layers;              /* backbone layers (32)                                  */
  int d_model;               /* backbone width (4096), a multiple of 128              */
  int n_heads;               /* attention heads (32)                                  */
  int head_dim;              /* head width, must be 128                               */
  int d_ff;                  /* SwiGLU hidden width (11008), a multiple of 64         */
  int n_new;                 /* tokens appended per vehicle and call, 1..8 (4)        */
  int max_batch;             /* largest B of any later call; n_new * max_batch <= 256 */
  long long max_cache_rows;  /* rows of every K/V cache buffer passed to fsx_append   */
  float rope_base;           /* rotary base (10000), > 1                              */
} fsx_append_config;

/* Host fp32 backbone weights, copied (and converted) by fsx_append_create;
 * every matrix is row-major [out_features, in_features], stacked over layers. */
typedef struct {
  const float* attn_norm;  /* [n_layers, d]                     RMSNorm gain, attention */
  const float* wq;         /* [n_layers, n_heads*head_dim, d]   W_q                     */
  const float* wk;         /* [n_layers, n_heads*head_dim, d]   W_k                     */
  const float* wv;         /* [n_layers, n_heads*head_dim, d]   W_v                     */
  const float* wo;         /* [n_layers, d, n_heads*head_dim]   W_o                     */
  const float* mlp_norm;   /* [n_layers, d]                     RMSNorm gain, SwiGLU    */
  const float* w_gate;     /* [n_layers, d_ff, d]               SwiGLU gate             */
  const float* w_up;       /* [n_layers, d_ff, d]               SwiGLU up               */
  const float* w_down;     /* [n_layers, d, d_ff]               SwiGLU down             */
} fsx_append_weights;

/* Create an append handle on `device`: validates cfg (host), uploads fp16
 * weights in the tensor-core tile order, allocates workspace for
 * cfg->max_batch vehicles. Blocking. Errors: INVALID_ARG (null pointers,
 * non-positive fields), UNSUPPORTED (shape outside the list above), OOM, CUDA. */
fsx_status fsx_append_create(const fsx_append_config* cfg, const fsx_append_weights* w, int device,
                             fsx_append_handle* out);

/* Append n_new tokens for each of B vehicles.
 *   k_cache, v_cache : HOST arrays of n_layers DEVICE pointers, none NULL; layer
 *                      l points to bf16 [max_cache_rows, n_heads, head_dim]
 *                      rows, token-major. Read, and written only at the rows
 *                      named by d_dst_rows.
 *   d_offsets        : DEVICE int64 [B+1], non-decreasing, offsets[0] >= 0,
 *                      offsets[B] <= max_cache_rows: vehicle b's cached tokens
 *                      0 .. L_b-1 are rows offsets[b] .. offsets[b+1]-1 (L_b may be 0).
 *   d_dst_rows       : DEVICE int64 [B]: vehicle b's new rows are written at rows
 *                      dst[b] .. dst[b] + n_new - 1 of every layer. These ranges
 *                      must lie in [0, max_cache_rows), must not overlap each
 *                      other, and must not overlap [offsets[0], offsets[B]).
 *   B                : 1 .. max_batch.
 *   d_x_new          : DEVICE bf16 [B, n_new, d] embeddings of the new tokens.
 *   d_hidden         : DEVICE fp32 [B, n_new, d] output: the residual stream
 *                      after the last layer (no final norm).
 * Enqueued on `stream` (kernel by kernel, no host synchronisation). The
 * device-side checks of offsets and destination rows set a sticky status read
 * by fsx_append_get_status; such a call writes no cache row and leaves d_hidden
 * undefined. A handle must not run two appends concurrently, and an append must
 * not run concurrently with a tick that reads the rows it writes. */
fsx_status fsx_append(fsx_append_handle h, void* const* k_cache, void* const* v_cache,
                      const int64_t* d_offsets, const int64_t* d_dst_rows, int B,
                      const void* d_x_new, float* d_hidden, void* stream);

/* Synchronises `stream`, then returns and clears the handle's device status
 * word (FSX_OK or FSX_ERR_DEVICE_ARG). */
fsx_status fsx_append_get_status(fsx_append_handle h, void* stream);

/* enable = 1: later appends on this handle run no kernel that waits on other CTAs
 * (the residual GEMMs are not split along K), so an append can share the GPU with a
 * tick whose single-launch kernel needs all of its CTAs resident (the concurrent
 * schedule of fsx_session). Slower per append; enable = 0 restores the default. */
fsx_status fsx_append_set_concurrent(fsx_append_handle h, int enable);

/* Bytes of the handle's fp16 weight arena (algorithmic weight bytes per call). */
long long fsx_append_weight_bytes(fsx_append_handle h);

/* Releases the handle's device memory (synchronises its device). */
void fsx_append_destroy(fsx_append_handle h);

/* ====================================================== the asynchronous fast-slow schedule
 * Sec. 3.3 and Fig. 1: the fast system ticks every 50 ms on the cache as it stands,
 * while every K = 4 ticks the slow system appends the newest frame's tokens behind
 * it. A session drives one vehicle's tick handle and append handle over one cache:
 * it owns the cache's committed length, gives every append the rows after everything
 * already reserved, and gives every tick a snapshot -- the rows of the appends that
 * have completed -- so a tick never reads a row that is being written and the
 * append-only cache needs no lock.
 *   FSX_SCHED_SERIAL     appends run on the tick stream: a tick waits for an append
 *                        in flight and reads its rows.
 *   FSX_SCHED_CONCURRENT appends run on a low-priority stream of their own, ticks on
 *                        a high-priority stream; the append handle is switched to
 *                        fsx_append_set_concurrent(h, 1), so no append kernel waits
 *                        on other CTAs and the single-launch tick always gets its SMs.
 * The session never frees the handles or the cache; destroy it before them. */
typedef struct fsx_session_s* fsx_session;
enum { FSX_SCHED_SERIAL = 0, FSX_SCHED_CONCURRENT = 1 };

/* tick: an fsx_handle whose max_total_cache_tokens >= capacity_rows (one vehicle);
 * append: an fsx_append_handle with the same n_layers and n_new tokens per call and
 * max_cache_rows >= capacity_rows; k_cache, v_cache: HOST arrays of n_layers DEVICE
 * pointers to bf16 [capacity_rows, n_heads, head_dim] buffers whose first
 * committed_rows rows hold the cache. Creates the session's two streams. */
fsx_status fsx_session_create(fsx_handle tick, fsx_append_handle append, void* const* k_cache, void* const* v_cache,
                              int n_layers, int n_new, long long capacity_rows, long long committed_rows, int mode,
                              int device, fsx_session* out);

/* Enqueue one append of n_new tokens (d_x_new: DEVICE bf16 [1, n_new, d_backbone])
 * at the rows after everything reserved so far, attending to all of them; the hidden
 * states go to d_hidden (DEVICE fp32 [1, n_new, d_backbone]). Asynchronous on the
 * session's append stream. FSX_ERR_INVALID_ARG when the rows would pass the capacity. */
fsx_status fsx_session_append(fsx_session s, const void* d_x_new, float* d_hidden);

/* Enqueue one tick (d_frames: DEVICE [1, n_frame, d] of the tick handle's frame dtype)
 * over the current snapshot on the session's tick stream; *snapshot_rows (if not NULL)
 * receives the number of cache rows the tick reads. */
fsx_status fsx_session_tick(fsx_session s, const void* d_frames, float* d_waypoints, long long* snapshot_rows);

/* Rows of completed appends (retires finished appends; does not block), and rows
 * reserved including appends in flight. */
long long fsx_session_committed(fsx_session s);
long long fsx_session_reserved(fsx_session s);
/* The session's tick and append streams (cudaStream_t), e.g. to time them. */
void* fsx_session_tick_stream(fsx_session s);
void* fsx_session_append_stream(fsx_session s);
/* Waits for every append and tick enqueued so far. */
fsx_status fsx_session_sync(fsx_session s);
void fsx_session_destroy(fsx_session s);

#ifdef __cplusplus
}
#endif
#endif /* FSX_H */
