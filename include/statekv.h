/*
 * statekv.h -- C ABI of the GB300 (sm_103a) StateKV per-frame cache-builder step.
 *
 * StateKV (Eyzaguirre, Wu, Niebles, "Linear Scaling Video VLMs for Long Video
 * Understanding") builds a video VLM's KV cache one frame at a time.  Per layer
 * it keeps two states (Sec. 3.2, Eq. 4):
 *   - the compressed state C (capacity B tokens), the only cross-frame context
 *     a new frame can attend to while the cache is built;
 *   - the detailed state D (every frame's K and V), used only for decoding.
 * For each new frame n and each layer (Sec. 3.3):
 *   (a1) the frame's T queries attend, GQA-style, to [C ; frame] (Eq. 5) with
 *        every state token visible and causal order inside the frame;
 *   (a2) fused with it, each pool token's importance -- the attention it
 *        receives, summed over the frame's queries (Eq. 1) and over the query
 *        heads of its KV head (App. A: sinks are kept per layer and KV head) --
 *        is recovered from the saved log-sum-exp (App. B.1);
 *   (a3) the B best-scoring tokens of the pool C + frame become the new C
 *        (Eq. 6); ties keep the older token;
 *   (a4) evicted state slots receive the admitted frame rows (bit copies);
 *   (a5) the frame's K and V are appended to D, and the virtual length
 *        L_n = n * T advances (Sec. 3.3, "virtual sequence length").
 *
 * Memory: the caller allocates one device arena (statekv_arena_bytes) and the
 * per-call input/output buffers.  The library never allocates device memory
 * and never frees caller memory.  Every call is asynchronous on the given
 * CUDA stream; argument errors are reported synchronously and enqueue nothing.
 *
 * Layouts (all row-major, bf16 = IEEE bfloat16, 16-byte aligned pointers):
 *   per-call Q      [stream_count][layer_count][T][Hq][d]
 *   per-call K, V   [stream_count][layer_count][T][Hkv][d]   (token-major)
 *   per-call out    [stream_count][layer_count][T][Hq][d]
 *   importance      fp32 [stream_count][layer_count][Hkv][B + T]
 * Query head h belongs to KV head h / (Hq / Hkv).  Token t of frame n (1-based)
 * sits at virtual position (n - 1) * T + t; rotary embeddings are expected to
 * be applied by the caller at those positions (Sec. 3.3).
 *
 * Threading: one host thread per handle.  Calls on one stream run in order.
 */
#ifndef STATEKV_H
#define STATEKV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* A cudaStream_t (struct CUstream_st*), declared here without CUDA headers.
 * NULL means the legacy default stream. */
typedef struct CUstream_st* statekv_stream;

typedef enum {
    STATEKV_OK = 0,
    STATEKV_ERR_INVALID_ARG = 1,     /* null/misaligned pointer, bad range or shape */
    STATEKV_ERR_UNSUPPORTED = 2,     /* valid but not built (e.g. head_dim not 64/128) */
    STATEKV_ERR_CACHE_FULL = 3,      /* a stream/layer already holds max_frames frames */
    STATEKV_ERR_CUDA = 4,            /* a CUDA runtime call failed */
    STATEKV_ERR_DEVICE_TIMEOUT = 5,  /* a kernel's bounded wait expired (sticky) */
    STATEKV_ERR_ARENA_TOO_SMALL = 6, /* arena smaller than statekv_arena_bytes() */
    STATEKV_ERR_DEVICE_FAULT = 7     /* a kernel detected an internal inconsistency (sticky) */
} statekv_status;

typedef struct statekv_handle statekv_handle;

typedef struct {
    int32_t num_streams;      /* independent videos sharing the handle (>= 1) */
    int32_t num_layers;       /* layers per stream (>= 1) */
    int32_t num_q_heads;      /* Hq */
    int32_t num_kv_heads;     /* Hkv, Hq % Hkv == 0 */
    int32_t head_dim;         /* d: 64 or 128 */
    int32_t tokens_per_frame; /* T >= 1 */
    int32_t state_capacity;   /* B >= 0 (B = 0: no cross-frame context) */
    int32_t max_frames;       /* decode-cache capacity per stream/layer, in frames */
    int32_t causal_in_frame;  /* 1: key t visible to query i iff t <= i (Eq. 5's M_n);
                                 0: every frame key visible (variant) */
    int32_t host_staging;     /* 1: reserve arena space (two frames) for the host-buffer calls */
    float softmax_scale;      /* 0 -> 1 / sqrt(head_dim) (Eq. 5) */
    uint32_t watchdog_ms;     /* bound on every device-side wait; 0 -> 2000 ms */
    int32_t selection;        /* which B tokens the state keeps after each frame:
                                 0 = the method's top-B importance (Eq. 6);
                                 1 = recency window, the B most recent tokens (the
                                     ReKV-style baseline the paper compares with);
                                     no importance is computed, so the per-call
                                     importance pointer must be NULL;
                                 2 = layer-level selection (App. A): one top-B per
                                     (stream, layer) by the importance summed over
                                     every KV head, applied to all KV heads, which
                                     then hold the same positions; the exported
                                     importance stays per KV head */
} statekv_config;

/* Bytes of device arena the configuration needs.  Returns INVALID_ARG or
 * UNSUPPORTED for a bad configuration. */
statekv_status statekv_arena_bytes(const statekv_config* cfg, size_t* bytes);

/* Creates a handle over a caller-owned device arena of at least
 * statekv_arena_bytes() bytes (256-byte aligned), whose prior contents do not
 * matter.  Zeroes the states and the decode caches (synchronously); every
 * stream/layer starts at frame 1 with an empty state.  The arena must outlive
 * the handle. */
statekv_status statekv_init(const statekv_config* cfg, void* device_arena, size_t arena_bytes,
                            statekv_handle** out);

typedef struct {
    int32_t stream_begin, stream_count; /* streams [begin, begin + count) */
    int32_t layer_begin, layer_count;   /* layers  [begin, begin + count) */
    const void* q;                      /* bf16, layout above (device) */
    const void* k;
    const void* v;
    void* out;                          /* bf16 attention output (device) */
    float* importance;                  /* nullable fp32 (device): per KV head, columns
                                           0..B-1 = state slots in their pre-call slot
                                           order (empty slots 0), columns B..B+T-1 =
                                           the frame's tokens */
} statekv_frame_args;

/* Processes the next frame of every (stream, layer) in the ranges: steps
 * (a1)-(a5) above.  Each covered (stream, layer) advances by one frame.
 * Returns CACHE_FULL (and enqueues nothing) if any of them already holds
 * max_frames frames, and DEVICE_TIMEOUT if an earlier call's kernel reported
 * an expired wait. */
statekv_status statekv_prefill_frame(statekv_handle* h, const statekv_frame_args* args,
                                     statekv_stream stream);

/* Exact full self-attention of the next frame, the comparison baseline of
 * Sec. 4.1 / App. B ("full SA"): for every query of the frame, softmax over
 * all tokens of the frames already processed (read from the decode cache,
 * every one visible) followed by the frame's own tokens (causal within the
 * frame as configured), times the matching values.  Writes out only: no
 * importance (args->importance must be NULL, else INVALID_ARG), and no change
 * to the states, the decode cache or the frame counters, so it can be timed
 * next to statekv_prefill_frame on the same handle ("given the preceding
 * cache, process one more frame").  Its cost grows with the frame index;
 * statekv_prefill_frame's does not. */
statekv_status statekv_full_attention_frame(statekv_handle* h, const statekv_frame_args* args,
                                           statekv_stream stream);

/* ---- App. A assumption diagnostics -------------------------------------
 * The paper validates its two assumptions on the full-attention baseline
 * (App. A): layer-level scores (attention summed over the frame's queries
 * within each head, then over every head of the layer), the concentration
 * C_{n,B} of historical attention in the top-B historical tokens (App. A.1),
 * and the candidate-pool recall, weighted recall, retention and churn of
 * consecutive top-B oracle states (App. A.2).  These calls compute the same
 * quantities on device buffers; ratios are the quotients of the sums they
 * return. */

/* Device workspace (bytes) statekv_full_attention_scores needs for a call
 * covering stream_count x layer_count (stream, layer) units: one fp32 partial
 * per (unit, KV head, 128-query tile, key slot of max_frames * T + T). */
statekv_status statekv_scores_workspace_bytes(const statekv_handle* h, int32_t stream_count,
                                              int32_t layer_count, size_t* bytes);

/* The exact full self-attention of the next frame, as
 * statekv_full_attention_frame (out written the same way, states, caches and
 * counters unchanged), plus App. A's layer-level score of every key:
 *   scores[u][j] = sum over every query head of the layer and every query of
 *                  the frame of the attention weight on key position j,
 * for j < L_n + T (the frames processed so far, then the frame's own tokens),
 * and 0 for j in [L_n + T, max_frames * T).
 *   scores     fp32 [stream_count][layer_count][max_frames * T] (device, 4-byte
 *              aligned)
 *   workspace  device memory (16-byte aligned) of at least
 *              statekv_scores_workspace_bytes() bytes; its contents are scratch
 * args->importance must be NULL.  INVALID_ARG for bad arguments or a covered
 * (stream, layer) that holds decoded tokens; CACHE_FULL if one already holds
 * max_frames frames (the scores row would not fit the next frame). */
statekv_status statekv_full_attention_scores(statekv_handle* h, const statekv_frame_args* args,
                                             float* scores, void* workspace,
                                             size_t workspace_bytes, statekv_stream stream);

/* Top-B membership (the T_{n,B} of App. A.1 and the oracle states S_n of
 * App. A.2): for each of `rows` rows, mask[r][j] = 1 for the min(B, n)
 * highest scores among scores[r][0 .. n) -- ties to the lower position j --
 * and 0 for every other j < row_stride.  Scores are attention sums, >= 0;
 * negative entries and NaN rank as 0.
 *   scores  fp32 [rows][row_stride] (device, 4-byte aligned)
 *   mask    uint8 [rows][row_stride] (device)
 * Needs 0 <= n <= row_stride <= 2^31 and B >= 0.  No handle: the call only
 * enqueues one kernel on `stream`. */
statekv_status statekv_topb_mask(const float* scores, int32_t rows, int64_t n, int64_t row_stride,
                                 int64_t B, uint8_t* mask, statekv_stream stream);

/* App. A.1 sums per row r (fp64 [rows][2], device):
 *   out[r][0] = sum of scores[r][j] over j < n with mask[r][j] != 0
 *   out[r][1] = sum of scores[r][j] over j < n
 * With n = L_n (historical keys only) and mask from statekv_topb_mask over the
 * same n, C_{n,B} = out[r][0] / out[r][1]. */
statekv_status statekv_concentration_sums(const float* scores, const uint8_t* mask, int32_t rows,
                                          int64_t n, int64_t row_stride, double* out,
                                          statekv_stream stream);

/* App. A.2 counts per row r (fp64 [rows][6], device), with
 *   S_n  = { j < n_seen : mask_n[r][j] }          (top-B of frame n's scores)
 *   S_n1 = { j < n_seen + T : mask_n1[r][j] }     (top-B of frame n+1's scores)
 *   P    = S_n plus the positions [n_seen, n_seen + T) of frame n+1
 *   w    = scores_n1[r]
 * out[r] = { |S_n1 & P|, |S_n1|, w(S_n1 & P), w(S_n1), |S_n & S_n1|, |S_n| }:
 * recall = out[0] / out[1], weighted recall = out[2] / out[3], retention =
 * out[4] / out[5], churn = (out[1] - out[4]) / out[1].  All three inputs are
 * [rows][row_stride] with n_seen + T <= row_stride. */
statekv_status statekv_state_metrics(const uint8_t* mask_n, const uint8_t* mask_n1,
                                     const float* scores_n1, int32_t rows, int64_t n_seen,
                                     int32_t T, int64_t row_stride, double* out,
                                     statekv_stream stream);

/* ---- Full per-frame transformer block ----------------------------------
 * One frame of every layer of a Qwen2-style decoder around the StateKV step,
 * layers in order (layer l + 1 reads layer l's output), per layer:
 *   h  = RMSNorm(x) * norm_attn
 *   [q k v] = h W_qkv^T + b_qkv;  q, k rotated by RoPE at the virtual
 *            positions L_n + t (Sec. 3.3: positions follow the virtual
 *            sequence length, not the cache size), with one RoPE scaling for
 *            the whole run (Sec. 3.3, "consistent RoPE scaling")
 *   o  = the StateKV step of statekv_prefill_frame on (q, k, v) (steps a1-a5:
 *        the layer's state and decode cache advance by one frame)
 *   x1 = x + o W_o^T
 *   x2 = x1 + (SiLU(h2 W_gate^T) * (h2 W_up^T)) W_down^T,  h2 = RMSNorm(x1) * norm_mlp
 * bf16 storage between steps, fp32 arithmetic.  The projections run on the
 * library's own tensor-core GEMMs: for up to 256 rows (one stream's frame) a
 * split-K kernel whose clusters add their partial sums in distributed shared
 * memory, with bias + RoPE, the residual add and SiLU * up in its epilogues;
 * above that a cooperative split-K kernel.  Weight matrices are row-major
 * [out features][in features] (torch.nn.Linear layout). */
typedef struct {
    int32_t hidden;            /* model width (multiple of 8, at most 8192) */
    int32_t intermediate;      /* MLP width (multiple of 8) */
    float rms_eps;             /* RMSNorm epsilon */
    float rope_theta;          /* RoPE base: pair k of head dim d turns at theta^(-2k/d) */
    float yarn_factor;         /* <= 1: plain RoPE; s > 1: YaRN scaling by s over a
                                  trained context of yarn_original_max tokens (pairs
                                  whose wavelength fits the context fewer than once
                                  turn s times slower, more than 32 times unchanged,
                                  linear in between; q and k scaled by 0.1 ln s + 1) */
    int32_t yarn_original_max;
} statekv_block_config;

typedef struct {
    const void* norm_attn;     /* bf16 [hidden] */
    const void* w_qkv;         /* bf16 [(Hq + 2 Hkv) d][hidden]: q, then k, then v rows */
    const void* b_qkv;         /* bf16 [(Hq + 2 Hkv) d], or NULL for no bias */
    const void* w_o;           /* bf16 [hidden][Hq d] */
    const void* norm_mlp;      /* bf16 [hidden] */
    const void* w_gate_up;     /* bf16 [2 intermediate][hidden]: gate rows, then up rows */
    const void* w_down;        /* bf16 [hidden][intermediate] */
} statekv_block_weights;

/* Device workspace (bytes, 256-byte aligned by the caller) for one
 * statekv_block_frame call over stream_count streams. */
statekv_status statekv_block_workspace_bytes(const statekv_handle* h,
                                             const statekv_block_config* bc,
                                             int32_t stream_count, size_t* bytes);

/* Runs the next frame of streams [stream_begin, stream_begin + stream_count)
 * through layers [layer_begin, layer_begin + layer_count) in order.
 *   weights  host array of num_layers entries (entry l for layer l; device
 *            pointers, each 16-byte aligned)
 *   x_in     bf16 [stream_count][T][hidden] (device): the frame's input to
 *            layer layer_begin; not modified
 *   x_out    bf16 [stream_count][T][hidden] (device): layer
 *            layer_begin + layer_count - 1's output (may equal x_in)
 * Every covered (stream, layer) advances by one frame.  The call only
 * enqueues work on `stream` (no synchronisation).  Errors as
 * statekv_prefill_frame, INVALID_ARG for a bad block config (head_dim / 2 >
 * 64 rotation pairs, sizes not multiples of 8, hidden > 8192) or a workspace
 * smaller than statekv_block_workspace_bytes(); nothing is enqueued on an
 * argument error, CUDA if a launch fails. */
statekv_status statekv_block_frame(statekv_handle* h, const statekv_block_config* bc,
                                   const statekv_block_weights* weights, int32_t stream_begin,
                                   int32_t stream_count, int32_t layer_begin, int32_t layer_count,
                                   const void* x_in, void* x_out, void* workspace,
                                   size_t workspace_bytes, statekv_stream stream);

/* Decoding over the detailed cache D_N (Sec. 3.2 / 3.3: decoding reads only
 * the detailed state; the compressed state is not used).  For every covered
 * (stream, layer), the num_tokens new tokens (a prompt, or one generated
 * token per call) attend to every row of the decode cache -- all video
 * frames processed so far, then the tokens of earlier decode calls -- and
 * causally to each other; afterwards their K/V rows are appended to the
 * cache.  q: bf16 [S_cnt][L_cnt][num_tokens][Hq][d]; k, v: bf16
 * [S_cnt][L_cnt][num_tokens][Hkv][d]; out: bf16 like q (all device, 16-byte
 * aligned).  Once a (stream, layer) has decoded tokens, statekv_prefill_frame
 * refuses it (INVALID_ARG): the video part is closed.  Returns CACHE_FULL if
 * the cache (max_frames * T rows per head) cannot take the new rows.
 * num_tokens must lie in [1, 4096]. */
typedef struct {
    int32_t stream_begin, stream_count;
    int32_t layer_begin, layer_count;
    int32_t num_tokens;
    const void* q;
    const void* k;
    const void* v;
    void* out;
} statekv_decode_args;

statekv_status statekv_decode_step(statekv_handle* h, const statekv_decode_args* args,
                                   statekv_stream stream);

/* Same step with HOST buffers (pinned memory recommended): q/k/v are copied
 * into the arena's staging area, the step runs, and out (and importance if
 * non-null) are copied back, all asynchronously on `stream`.  Host buffers
 * must stay valid until the stream is synchronised.  Needs host_staging = 1. */
statekv_status statekv_prefill_frame_host(statekv_handle* h, const statekv_frame_args* args,
                                          statekv_stream stream);

/* n consecutive frames (Sec. 3.3's per-frame step, n times) from HOST
 * buffers, with the copies pipelined against the steps: frames[i] holds the
 * host q/k/v/out (and importance, or null) of frame i, laid out as in
 * statekv_prefill_frame_host.  Every entry must cover the same streams and
 * layers, and either every entry or none has an importance buffer.  The
 * arena's staging area holds two frames; frame i + 1 is copied in on an
 * internal copy stream while frame i runs on `stream`, and frame i - 1 is
 * copied out on another.  Ordering: the first copy waits for the work
 * already enqueued on `stream`, and `stream` waits for the last copy out, so
 * the results are in the host buffers once `stream` is synchronised.  Host
 * buffers must stay valid (and the inputs unchanged) until then.  Returns
 * CACHE_FULL (with no work enqueued) if a covered (stream, layer) cannot take
 * n more frames.  Needs host_staging = 1. */
statekv_status statekv_prefill_frames_host(statekv_handle* h, const statekv_frame_args* frames,
                                           int32_t n, statekv_stream stream);

typedef struct {
    const void* k;            /* bf16 [Hkv][B][d] (device); slot order is arbitrary */
    const void* v;            /* bf16 [Hkv][B][d] (device) */
    const int32_t* positions; /* int32 [Hkv][B] (device); virtual position, -1 = empty */
    int32_t count;            /* valid slots per KV head: min(B, frames * T) */
    int32_t frames;           /* frames processed */
    int64_t virtual_len;      /* L_n = frames * T */
} statekv_state_info;

typedef struct {
    const void* k;            /* bf16 [Hkv][capacity][d] (device) */
    const void* v;
    int64_t length;           /* rows written: frames * T + decoded tokens */
    int64_t capacity;         /* max_frames * T */
} statekv_cache_info;

/* Borrowed device pointers into the arena, valid until statekv_destroy.  The
 * contents are current once the stream of the last prefill call is
 * synchronised; the counters are host-side and current immediately.
 *
 * statekv_state_view: the compressed state of one (stream, layer) -- Sec. 3.3,
 * Eq. 6's S_n, the B tokens per KV head kept by the top-B selection, with
 * their virtual positions (Sec. 3.3: token t of frame n sits at (n-1) T + t)
 * and the virtual length L_n.  Errors: INVALID_ARG for a null handle or
 * output, or a (stream, layer) outside the configuration. */
statekv_status statekv_state_view(const statekv_handle* h, int32_t stream, int32_t layer,
                                  statekv_state_info* out);
/* statekv_cache_view: the detailed state of one (stream, layer) -- Sec. 3.2,
 * Eq. 4's D_n, every frame's K/V rows appended in order (then any decoded
 * tokens), which decoding attends to.  Errors: INVALID_ARG for a null handle
 * or output, or a (stream, layer) outside the configuration. */
statekv_status statekv_cache_view(const statekv_handle* h, int32_t stream, int32_t layer,
                                  statekv_cache_info* out);

/* Optional per-kernel timing with CUDA events recorded on the call's stream
 * around each launch.  enable != 0 starts a new record; read synchronises on
 * the recorded events and returns, per kernel kind (0 = decode-cache append,
 * 1 = frame attention + importance, 2 = state select/gather, 3 = the block's
 * projection GEMMs, 4 = the block's RMSNorm / RoPE / SiLU kernels), the
 * number of launches and their summed device milliseconds. */
typedef struct {
    int64_t launches[5];
    double milliseconds[5];
} statekv_profile;
statekv_status statekv_profile_enable(statekv_handle* h, int32_t enable);
statekv_status statekv_profile_read(statekv_handle* h, statekv_profile* out);

/* Synchronises the device and reports a device error (DEVICE_TIMEOUT or
 * DEVICE_FAULT) if a kernel recorded one. */
statekv_status statekv_sync(statekv_handle* h);

/* Failure-detection self-test.  Enqueues the frame-attention kernel for one
 * work unit whose producer first waits on a barrier that nothing completes:
 * the wait expires after half the handle's watchdog (watchdog_ms), before
 * any other wait can, the kernel records DEVICE_TIMEOUT in the status word
 * (site 1) and every warp leaves
 * through its own bounded wait; no input is read and no copy or MMA is
 * issued.  The handle's status is sticky afterwards, so the next call (e.g.
 * statekv_sync) returns STATEKV_ERR_DEVICE_TIMEOUT; use a handle made for
 * the test.  The GPU context stays usable. */
statekv_status statekv_watchdog_selftest(statekv_handle* h, statekv_stream stream);

/* The raw device status word (0 = none): low byte 1 = an attention-kernel
 * wait expired (bits 8..15 name the waiting site), 2 = the selection kernel
 * found an inconsistent top-B split, 3 = a projection-GEMM wait expired,
 * 4 = a decode-kernel wait expired, 5 / 6 = a debug build's bounds check or
 * guard band failed (see statekv_debug_check).  Read without synchronising. */
statekv_status statekv_device_error(const statekv_handle* h, int32_t* code);

/* Debug builds (the library compiled with STATEKV_DEBUG_CHECKS=1, e.g.
 * build_ext.build(debug=True) -> libstatekv_debug.so) put a 256-byte guard band
 * after every arena region, filled with 0xA5 at init, and check indices before
 * the state, cache and importance writes; a failed check records a bounds
 * fault in the status word and skips the access (no trap).  This call
 * enqueues a comparison of every guard byte with its fill on `stream`; an
 * overwritten band records a canary fault.  Either fault is reported, like any
 * device fault, as STATEKV_ERR_DEVICE_FAULT by the next call that reads the
 * status (statekv_sync), with the kind in statekv_device_error's low byte
 * (5 bounds, 6 canary) and the site or band in bits 8..15.  A release build
 * returns STATEKV_ERR_UNSUPPORTED and enqueues nothing.  These are the
 * sanitizer substitutes of the implementation; the paper has no counterpart. */
statekv_status statekv_debug_check(statekv_handle* h, statekv_stream stream);

/* Frame attention with importance (steps a1 and a2) for ONE (stream, layer)
 * against a caller-given state, for callers that cannot allocate device
 * memory -- e.g. plugins held to a host application's memory budget, or code
 * that must not call cudaMalloc while another component captures a stream.
 * The paper has no counterpart: this is a packaging of the same kernel.
 * Its scratch (importance partials, per-head counts, a status word) is a
 * fixed set of file-scope device arrays, resident on every GPU that loads the
 * library until the process exits: at most 2^20 fp32 partials, i.e.
 * num_kv_heads * ceil(G * T / 128) * (B + T) <= 1048576 with G = Hq / Hkv, and
 * num_kv_heads <= 64; larger shapes return STATEKV_ERR_UNSUPPORTED.  The call
 * allocates nothing.  Its first call on a device looks up the arrays' device
 * addresses; make that first call before any stream capture.  Calls share the
 * scratch: calls that overlap on the GPU race.  The call synchronises `stream`
 * before it returns and reports its own DEVICE_TIMEOUT, so `stream` must not
 * be under capture (STATEKV_ERR_INVALID_ARG, nothing enqueued); while another
 * component captures, pass a cudaStreamNonBlocking stream, since a blocking
 * stream (the legacy default stream among them) synchronises implicitly with
 * the capturing one and so invalidates that capture.  T above 4096, more than
 * 64 KV heads or G * T above 2^31 - 1 also return STATEKV_ERR_UNSUPPORTED.
 *   cfg           num_q_heads, num_kv_heads, head_dim, tokens_per_frame,
 *                 state_capacity (B), causal_in_frame, softmax_scale,
 *                 watchdog_ms are used; the rest is ignored
 *   q, k, v       bf16 [T][Hq][d], [T][Hkv][d], [T][Hkv][d] (device)
 *   state_k/v     bf16 [Hkv][B][d] (device); rows [0, state_count) are valid;
 *                 the rows after them, up to the next multiple of 128 (or B),
 *                 are read by the last key tile and must hold finite values
 *                 (zeros, say): their weights are 0, but 0 times NaN is NaN
 *   out           bf16 [T][Hq][d] (device)
 *   importance    fp32 [Hkv][B + T] (device), columns as in statekv_frame_args
 * Nothing of the handle-based state is read or written. */
statekv_status statekv_frame_attention_noalloc(const statekv_config* cfg, const void* q,
                                               const void* k, const void* v, const void* state_k,
                                               const void* state_v, int32_t state_count,
                                               void* out, float* importance,
                                               statekv_stream stream);

void statekv_destroy(statekv_handle* h);
const char* statekv_status_string(statekv_status s);

#ifdef __cplusplus
}
#endif

#endif /* STATEKV_H */
