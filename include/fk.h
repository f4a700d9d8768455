/*
 * fk.h -- C ABI of the Forcing-KV hot path (hybrid KV-cache compression plus chunk
 * attention over the compressed cache) on one NVIDIA GB300 (sm_103a).
 *
 * The operations follow the paper's statement of the method:
 *   - static heads attend to [sink frames, transition-anchor frame, current chunk]
 *     (Sec. 4.2, Eq. 2);
 *   - dynamic heads score each history frame t against frame t+1 segment by segment
 *     with a cosine similarity, keep the floor(b*n) lowest-similarity segments of the
 *     n equal segments of each frame (BottomK, Sec. 4.3, Eq. 3; b = 1 - r, the keep
 *     budget, App. H) and attend to [sink, kept segments, anchor frame, current chunk]
 *     (Sec. 4.3, Eq. 4; the anchor is kept because a dynamic head's cache holds
 *     everything a static head keeps, Sec. 5.3);
 *   - compression starts once adjacent history frames exist (App. H); sink frames are
 *     never scored or evicted.
 *
 * Conventions shared by every call:
 *   - Tensors K, V, Q, O are bf16, token-major [tokens][n_heads][head_dim], row-major
 *     and contiguous ("the [seq, heads, dim] layout"), 16-byte aligned.
 *   - A tensor pointer may be device memory or host memory (pinned or pageable).  Host
 *     inputs are copied into library-owned device staging buffers on `stream`; a host output
 *     is written by an asynchronous device-to-host copy on `stream`, so the caller
 *     synchronizes `stream` before reading it (with fk_set_host_overlap on, the copies run on
 *     the handle's copy streams instead; see there).  Caller-owned device inputs must
 *     stay valid until the work queued on `stream` by the call has run.
 *   - `stream` is a cudaStream_t passed as void* (NULL = the legacy default stream).
 *   - Frames are numbered globally from 0 in append order.  The history is every frame
 *     appended before the current chunk; the current chunk is frames nh..nh+C-1, where
 *     nh is the number of history frames.  Segment id of segment j of frame t is t*n+j.
 *   - Every call returns a status code.  The library never aborts, traps or prints.
 *     Conditions found on the device (the scoring precondition, an expired bounded
 *     wait) are recorded in a device status word and reported by fk_sync_status.
 *   - The library owns all of its device memory; it is allocated in fk_create and
 *     released in fk_destroy.  No other call allocates.
 *   - A handle is not thread-safe: calls on one handle are made from one host thread.
 */
#ifndef FK_H
#define FK_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define FK_API __attribute__((visibility("default")))
#else
#define FK_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum fk_status {
  FK_OK = 0,
  FK_ERR_CONFIG = 1,   /* invalid configuration (see fk_config)                         */
  FK_ERR_ARG = 2,      /* null or misaligned pointer, layer/head out of range, short buffer */
  FK_ERR_STATE = 3,    /* call out of order: attend before compress, no current chunk,
                          layers out of step under layer-0 pooled scoring               */
  FK_ERR_FULL = 4,     /* unbounded window and max_history_frames would be exceeded      */
  FK_ERR_RANGE = 5,    /* scoring precondition violated: a token's squared key norm > 2^23 */
  FK_ERR_TIMEOUT = 6,  /* a bounded wait inside a kernel expired; outputs are undefined   */
  FK_ERR_CUDA = 7,     /* a CUDA runtime/driver call failed (no device, launch failure)   */
  FK_ERR_NOMEM = 8     /* device memory for the cache could not be allocated             */
} fk_status;

/* Selection scope of BottomK (Eq. 3). */
enum {
  FK_SCOPE_PER_FRAME = 0, /* keep floor(b*n) segments of every scoreable frame            */
  FK_SCOPE_POOLED = 1     /* keep floor(b*|T|*n) segments over all scoreable frames T      */
};

/* Which keys score the dynamic heads (Eq. 3). */
enum {
  FK_SCORE_PER_HEAD = 0,      /* each dynamic head scores its own keys                     */
  FK_SCORE_LAYER0_POOLED = 1  /* keys of every head of layer 0, pooled, score every dynamic
                                 head of every layer (the first block's keys stand in
                                 for every layer, Sec. 4.3); one kept set is shared by all
                                 dynamic heads                                              */
};

/* Which segments of a scoreable frame dynamic heads keep.  SIMILARITY is the method (Eq. 3);
 * the others are the paper's comparison rules, run through the same selection, compaction
 * and attention for speed comparisons (App. H and Sec. 5.3): ALL keeps every segment (with
 * n_sink_frames = 3 and window_frames = 4 on all-dynamic heads: the frame-level StreamingLLM
 * baseline; on neighbour heads with window_frames = L: Dummy Forcing), UNIFORM keeps the k
 * segments j = floor(i n / k), i < k (with n_segments = tokens_per_frame: uniform token
 * pruning), RANDOM keeps the k segments with the smallest seeded SplitMix64 values (random
 * token pruning).  k = floor(b n) as for SIMILARITY (n for ALL). */
enum {
  FK_SELECT_SIMILARITY = 0,
  FK_SELECT_ALL = 1,
  FK_SELECT_UNIFORM = 2,        /* per-frame scope only */
  FK_SELECT_RANDOM = 3
};

/* Operand precision of the chunk attention (the paper's quantization appendix: FP8 attention
 * on the compressed cache).  BF16: Q, K, V in bf16 (the method).
 * FP8_QK: Q K^T on OCP FP8 E4M3 operands with f32 accumulation; P V stays bf16.  Keys are
 * rounded to E4M3 unscaled (E4M3 keeps the same relative precision over its normal range,
 * 2^-6 to 448): FP8_QK requires key elements within +-448, larger ones saturate.  Each query
 * row (token, head) is scaled by 2^-e, e the smallest integer with max |q| <= 448 * 2^e, and
 * the logits are scaled back by 2^e, so the E4M3 rounding (to nearest, ties to even) is the
 * only inexact step before the softmax.  fk_quantize_e4m3 applies the same rounding.
 * FP8: Q K^T as FP8_QK, and P V on E4M3 operands too, f32 accumulation: values are rounded to
 * E4M3 unscaled (elements within +-448), and each softmax numerator exp(l - m) is scaled by
 * 2^6 before its E4M3 rounding, m being the running row maximum, which lags the row maximum by
 * at most a factor 2 (so a numerator stays within 2^7); the row normaliser is the sum of the
 * unrounded scaled numerators.  Both FP8 precisions require head_dim 128. */
enum {
  FK_ATTN_BF16 = 0,
  FK_ATTN_FP8_QK = 1,
  FK_ATTN_FP8 = 2
};

/* Configuration of one cache.  The method's quantities (Sec. 4.2-4.3 and App. H): F tokens per
 * frame and C frames per chunk (Eq. 2: the current chunk is tokens iCF..(i+1)CF-1); the sink
 * frames preserved at the start of the video (App. H); n segments per frame and the keep budget
 * b = 1 - r of dynamic heads (App. H sets n = 6, r = 0.3; Eq. 3 keeps the floor(b n) lowest-
 * similarity segments); the static/dynamic head map produced by offline head profiling (Sec. 4.1,
 * Eq. 1).  The remaining fields choose this library's execution (window capacity, selection
 * scope and proxy, incremental scoring, device, the paper's comparison rules, FP8). */
typedef struct fk_config {
  int32_t n_layers;             /* 1..256                                                  */
  int32_t n_heads;              /* 1..128                                                  */
  int32_t head_dim;             /* 64 or 128                                               */
  int32_t tokens_per_frame;     /* F >= 1, a multiple of n_segments (Eq. 2, App. H)        */
  int32_t frames_per_chunk;     /* C >= 1 (Eq. 2)                                          */
  int32_t n_sink_frames;        /* S >= 0: frames 0..S-1 are sinks, never evicted (App. H) */
  int32_t window_frames;        /* W >= 0 non-sink history frames kept, anchor included;
                                   0 = unbounded (capacity max_history_frames); the model's
                                   own attention window (App. H)                           */
  int32_t n_segments;           /* n >= 1 contiguous equal segments per frame (App. H)     */
  int32_t keep_budget_permille; /* b*1000 in [0, 1000]; k = floor(b*n) kept per frame
                                   (Eq. 3 with b = 1 - r; App. H: r = 0.3)                */
  int32_t select_scope;         /* FK_SCOPE_*                                              */
  int32_t score_source;         /* FK_SCORE_* (Sec. 4.3: the first block's keys as proxy)  */
  int32_t incremental;          /* 1: fk_compress scores only frame pairs not scored yet
                                   (a frame's pairs never change once both frames exist);
                                   0: every fk_compress rescores the whole window         */
  int32_t max_history_frames;   /* history capacity in frames, sinks included, when W = 0 */
  int32_t device;               /* CUDA device ordinal                                     */
  const uint8_t* head_is_static;/* host [n_layers*n_heads]: 1 = static head, 0 = dynamic
                                   (the classification of Sec. 4.1, Eq. 1); copied by
                                   fk_create                                               */
  int32_t selection;            /* FK_SELECT_* (0 = the method)                            */
  uint32_t select_seed;         /* seed of FK_SELECT_RANDOM                                */
  int32_t static_drop_anchor;   /* 1: static heads keep sink + current chunk only (Dummy
                                   Forcing's local heads); 0: sink + anchor + current (Eq. 2) */
  int32_t attn_precision;       /* FK_ATTN_* (0 = bf16)                                    */
} fk_config;

typedef struct fk_handle fk_handle;

/* Host-only validation of a configuration (no CUDA call).  FK_OK or FK_ERR_CONFIG /
 * FK_ERR_ARG.  fk_create runs the same checks first. */
FK_API fk_status fk_validate_config(const fk_config* cfg);

/* Create a cache on cfg->device and allocate all of its device memory: per head the packed
 * view of its key set (Eq. 2 for static heads, Eq. 4 plus the anchor for dynamic heads) and,
 * for dynamic heads, the history pages that scoring reads (the paper keeps history frames for
 * similarity computation, Sec. 5.2).  *out receives the handle (NULL on failure).  Errors:
 * FK_ERR_CONFIG / FK_ERR_ARG as fk_validate_config, FK_ERR_CUDA (no device, kernel setup),
 * FK_ERR_NOMEM (allocation). */
FK_API fk_status fk_create(const fk_config* cfg, fk_handle** out);

/* Release the handle and its device memory (synchronizes the device first). NULL is a no-op. */
FK_API void fk_destroy(fk_handle* h);

/* Append n_frames frames to the history of `layer` (e.g. loading sink and history
 * frames).  If a current chunk exists it first joins the history, and afterwards no
 * current chunk exists.  K, V: [n_frames*F][H][D].  Static heads keep only sink frames
 * and the newest non-sink frame (the anchor); dynamic heads keep every window frame
 * for scoring.  Marks the layer for fk_compress.  FK_ERR_FULL if the history would
 * exceed max_history_frames with W = 0. */
FK_API fk_status fk_append_frames(fk_handle* h, int layer, const void* K, const void* V, int n_frames,
                           void* stream);

/* Start AR step: the current chunk (if any) joins the history and K, V [C*F][H][D]
 * become the current chunk of `layer` (Eq. 2 and Eq. 4 K_{iCF:(i+1)CF}).  Marks the
 * layer for fk_compress. */
FK_API fk_status fk_append_chunk(fk_handle* h, int layer, const void* K, const void* V, void* stream);

/* Overwrite the current chunk's K, V [C*F][H][D] of `layer` (next denoising step of
 * the same AR step), or set it when none exists.  The history is unchanged. */
FK_API fk_status fk_set_current(fk_handle* h, int layer, const void* K, const void* V, void* stream);

/* Compress every layer marked by an append: score the new (or, with incremental = 0,
 * all) adjacent frame pairs of the window segment by segment (Eq. 3), select the kept
 * segments (BottomK, ties to the lower segment id) and compact each dynamic head's
 * keys and values into its packed view [current chunk | sinks | anchor | kept segments]
 * (attention does not depend on the order of the keys).
 * With no scoreable frame it only rebuilds the views.  Asynchronous on `stream`;
 * FK_ERR_STATE when layer-0 pooled scoring finds layers with different histories. */
FK_API fk_status fk_compress(fk_handle* h, void* stream);

/* O [C*F][H][D] = per head softmax(Q K^T / sqrt(D)) V over the head's key set: Eq. 2
 * for static heads, Eq. 4 plus the anchor frame for dynamic heads.  Q: [C*F][H][D].
 * Under FK_ATTN_FP8_QK, Q K^T runs on E4M3 operands (the rounding described there; P V in
 * bf16); under FK_ATTN_FP8 P V too.  FK_ERR_STATE if `layer` has no current chunk or was appended to since the last
 * fk_compress. */
FK_API fk_status fk_attend(fk_handle* h, int layer, const void* Q, void* O, void* stream);

/* Bytes of device memory currently holding live cache state: retained history pages,
 * the used part of every packed view (current chunk included), scores and kept lists.  The
 * cache-memory figure of Sec. 5.2 (KV memory of the compressed cache; the paper notes that
 * dynamic heads also keep history frames for similarity computation, counted here). */
FK_API size_t fk_cache_bytes(const fk_handle* h);

/* Bytes of device memory the handle allocated (all buffers, live or not). */
FK_API size_t fk_reserved_bytes(const fk_handle* h);

/* Number of keys head (layer, head) attends to at the current state (host-known). */
FK_API fk_status fk_key_count(const fk_handle* h, int layer, int head, int* n_keys);

/* Kept segment ids (t*n + j, ascending) of dynamic head (layer, head) after the last
 * fk_compress: the index set I_keep of Eq. 3 (Sec. 4.3); *n_out = 0 for a static head.  `out`
 * is caller-owned host memory of `capacity` ints.  Synchronizes `stream`.  FK_ERR_ARG if
 * capacity is too small (then *n_out holds the required count). */
FK_API fk_status fk_get_kept(fk_handle* h, int layer, int head, int32_t* out, int capacity, int* n_out,
                      void* stream);

/* Segment scores s_t^(j) (fp32, Eq. 3 under the score contract) of the scoreable
 * frames of dynamic head (layer, head): out[(t - *first_frame)*n + j] for the
 * *n_frames frames t = *first_frame .. .  Synchronizes `stream`. */
FK_API fk_status fk_get_scores(fk_handle* h, int layer, int head, float* out, int capacity,
                        int* first_frame, int* n_frames, void* stream);

/* Synchronize `stream` and report (then clear) device-side conditions:
 * FK_ERR_RANGE, FK_ERR_TIMEOUT, or FK_OK. */
FK_API fk_status fk_sync_status(fk_handle* h, void* stream);

/* Kernel timing: when enabled, every kernel launch is bracketed by CUDA events on its
 * stream.  fk_profile_read synchronizes and returns, per kernel kind, the total device
 * milliseconds and the number of launches since the last reset. */
enum { FK_KERNEL_APPEND = 0, FK_KERNEL_SCORE = 1, FK_KERNEL_SELECT = 2, FK_KERNEL_COMPACT = 3,
       FK_KERNEL_ATTEND = 4, FK_KERNEL_KINDS = 5 };
FK_API fk_status fk_profile_enable(fk_handle* h, int on);
FK_API fk_status fk_profile_read(fk_handle* h, int kind, double* total_ms, int64_t* launches);
FK_API fk_status fk_profile_reset(fk_handle* h);

/* Host-transfer overlap.  Off (the default): a host input (K, V of fk_append_chunk /
 * fk_set_current, Q of fk_attend) is copied into staging on `stream`, in call order, and a
 * host output (O of fk_attend) is copied back on `stream`.  On: a host input is copied at once
 * on a copy stream owned by the handle, into one of two staging slots per input kind, so the
 * copy overlaps the work already queued on `stream` (the kernel that reads it waits for the
 * copy; the next copy into a slot waits for the kernel that read it before); and a host
 * output is copied back on a second copy stream of the handle after the attention kernel, so
 * it overlaps the work queued after the call.  With overlap on, the caller guarantees that a
 * host input is final when the call is made (written by the CPU, not by device work still
 * pending on any stream) and unchanged until `stream` has run the call's work, and reads a
 * host output only after fk_wait_outputs (or fk_sync_status) on `stream` and a
 * synchronization of `stream`.  FK_ERR_ARG for a null handle. */
FK_API fk_status fk_set_host_overlap(fk_handle* h, int on);

/* Make `stream` wait for every host-output copy still pending on the handle's copy stream
 * (host overlap on); a no-op otherwise.  FK_ERR_ARG for a null handle. */
FK_API fk_status fk_wait_outputs(fk_handle* h, void* stream);

/* Failure-detection self-test (no counterpart in the paper): launches a one-thread kernel
 * that waits, with the same bounded-wait primitive as the hot-path kernels, on an mbarrier
 * that nothing completes; after limit_us microseconds (1..2,000,000) the wait gives up and
 * records the expiry in the handle's status word, so the next fk_sync_status returns
 * FK_ERR_TIMEOUT and clears it.  No fault: the CUDA context stays usable.  Asynchronous on
 * `stream`.  FK_ERR_ARG for a null handle or a limit out of range. */
FK_API fk_status fk_wait_selftest(fk_handle* h, int limit_us, void* stream);

/* HBM calibration (no counterpart in the paper): reads `bytes` of device memory once with
 * 16-byte streaming loads from a grid of 8 CTAs per SM and does nothing else.  Timed with CUDA
 * events like the hot-path kernels, its duration is the practical floor for any single launch
 * that must read that many bytes (it includes the launch and the first accesses' latency),
 * which the benchmark reports beside the HBM-bound kernels' fractions of the copy bandwidth.
 * src: device memory, 16-byte aligned; bytes: a multiple of 16 (0: no launch).  FK_ERR_ARG for
 * null, misaligned or host pointers.  Asynchronous on `stream`; allocates nothing. */
FK_API fk_status fk_stream_read(const void* src, size_t bytes, void* stream);

/* Kernels launched by this handle since creation (all kinds). */
FK_API int64_t fk_launch_count(const fk_handle* h);

/* Segment scores of consecutive frames of one head without allocating any memory.
 * The paper has no counterpart: this is a service entry point of this library.  It is for
 * callers that must not call cudaMalloc: code running inside a framework whose allocator owns
 * all device memory, or a real-time generation loop whose memory budget is fixed up front and
 * that cannot risk an allocation failing or stalling mid-stream.
 * K: device memory [n_frames][tokens_per_frame][head_dim] bf16 (one head's frames, oldest
 * first, 16-byte aligned).  scores: device memory [n_frames - 1][n_segments] fp32; on
 * completion scores[t][j] = s_t^(j), the cosine of segment j of frames t and t+1 (Eq. 3) under
 * the same score contract as fk_compress, bit-identical to fk_get_scores for the same frames.
 * status: NULL, or a caller-owned device int that the caller zeroes; the kernels OR into it the
 * conditions fk_sync_status would report for a handle: 1 when a token's contract squared key
 * norm exceeds 2^23 (the condition of FK_ERR_RANGE: the scores are then unspecified) and 2 when
 * a bounded device wait expired (the condition of FK_ERR_TIMEOUT: the scores are undefined).
 * With status NULL these conditions go unreported.
 * Limits: head_dim 64 or 128, 2 <= n_frames <= 256, 1 <= n_segments <= 32, n_frames *
 * n_segments <= 4096, tokens_per_frame a multiple of n_segments; larger sizes return
 * FK_ERR_CONFIG; host, null (K, scores) or misaligned pointers FK_ERR_ARG.  The scratch is one
 * fixed 65,728-byte array per device that loads the library (held until the process exits),
 * shared by every call and holding the last call's contents (each call clears what must start
 * at zero): calls whose work overlaps on the GPU (e.g. on two streams) race and must be ordered
 * by the caller.  The first call on a device resolves that array's address and must come before
 * any stream capture.  Asynchronous on `stream`; uses the current device. */
FK_API fk_status fk_segment_scores_noalloc(const void* K, int n_frames, int tokens_per_frame,
                                           int head_dim, int n_segments, float* scores,
                                           int* status, void* stream);

/* Offline head profiling (Sec. 4.1, Eq. 1): attention mass per key class.
 * Q: device [n_queries][n_heads][head_dim] bf16, the queries of the generated chunk.
 * K: device [n_keys][n_heads][head_dim] bf16, every key of the attention window in the order
 *    [generated chunk (n_generate) | sink frames (n_sink) | other history | transition frame
 *    (n_transition, the last frame before the chunk)]; both 16-byte aligned, token-major.
 * For every head h and query row, the softmax over all n_keys keys (scale 1/sqrt(head_dim))
 * is split by key class; the row's fractions are summed over the rows and ADDED to
 * mass[h][0..3] = {A_Total (= rows), A_Generate, A_Transition, A_Sink} (device, double; the
 * caller zeroes it, so repeated calls accumulate over steps).  A bounded device wait that
 * expires ORs the value 2 into *status (device int, caller-owned, zeroed by the caller).
 * Errors: FK_ERR_ARG for null, unaligned or host pointers; FK_ERR_CONFIG for head_dim not 64
 * or 128, n_heads outside 1..128, empty Q or K, or class counts exceeding n_keys.
 * Asynchronous on `stream`; allocates nothing; uses the current device. */
FK_API fk_status fk_head_profile(const void* Q, const void* K, int n_queries, int n_keys,
                                 int n_heads, int head_dim, int n_generate, int n_sink,
                                 int n_transition, double* mass, int* status, void* stream);

/* Eq. 1 on host-side masses ([n_heads][4] as written by fk_head_profile): head h is static
 * (head_is_static[h] = 1) when (A_Generate + A_Transition) / (A_Total - A_Sink) exceeds
 * alpha_permille / 1000 (alpha = 0.8 in the paper: 800), else dynamic (0).  A head with all
 * of its mass on the sink frames (A_Total - A_Sink <= 0) is static.  FK_ERR_ARG for null
 * pointers, FK_ERR_CONFIG for alpha outside 0..1000. */
FK_API fk_status fk_classify_heads(const double* mass, int n_heads, int alpha_permille,
                                   uint8_t* head_is_static);

/* E4M3 quantization of bf16 rows, as the FP8_QK attention applies it (see FK_ATTN_FP8_QK).
 * X: device [rows][dim] bf16; q8: device [rows][dim] bytes, OCP FP8 E4M3 codes; both 16-byte
 * aligned.  row_scaled = 1 (queries): row r is multiplied by 2^-e_r, e_r the smallest integer
 * with max_c |X[r][c]| <= 448 * 2^e_r (0 for an all-zero row; clamped to [-120, 120]), then
 * rounded to the nearest E4M3 value (ties to even, saturating at +-448); exps (device int8
 * [rows]) receives e_r.  row_scaled = 0 (keys): every element is rounded unscaled and exps may
 * be NULL.  dim: 64 or 128 when row_scaled, else a multiple of 8 from 8 to 1024; rows >= 0.
 * FK_ERR_ARG for null, unaligned or host pointers, FK_ERR_CONFIG for sizes out of range.
 * Asynchronous on `stream`; allocates nothing; uses the current device. */
FK_API fk_status fk_quantize_e4m3(const void* X, int64_t rows, int dim, int row_scaled,
                                  void* q8, int8_t* exps, void* stream);

/* Static text for a status code. */
FK_API const char* fk_status_str(fk_status s);

/* ABI version of this header: 4 (fk_config gained selection, select_seed and
 * static_drop_anchor after head_is_static in version 2, attn_precision in version 3;
 * fk_segment_scores_noalloc gained its status argument in version 4). */
FK_API int fk_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* FK_H */
