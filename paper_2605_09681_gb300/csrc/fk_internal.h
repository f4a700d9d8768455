// Internal declarations of the Forcing-KV library: handle state, kernel argument
// blocks and launchers.  Shared by the library's translation units only.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdint>
#include <vector>

#include "fk.h"

namespace fk {

using bf16 = __nv_bfloat16;

constexpr int kMaxHeads = 128;
constexpr int kMaxLayers = 256;
constexpr int kAttnBM = 128;          // query rows per attention CTA
constexpr int kAttnBN = 128;          // keys per attention tile
constexpr int kViewAlignRows = 128;   // packed views are padded to whole key tiles
// scoring CTA: 4 warps; a token is owned by 4 lanes, so a CTA covers 32 tokens of a segment
// (one frame-chunk)
constexpr int kScoreThreads = 128;
constexpr int kScoreTokensPerCta = (kScoreThreads / 32) * 8;

// device status word bits (set by kernels, read by fk_sync_status)
constexpr int kStatusRange = 1;
constexpr int kStatusTimeout = 2;

#ifdef __CUDACC__
// OCP FP8 E4M3 rounding of the FP8_QK attention (hardware cvt.rn.satfinite: to nearest, ties
// to even, saturating at +-448): two floats -> two codes, `lo` in the low byte
__device__ __forceinline__ uint32_t e4m3x2(float lo, float hi) {
  uint16_t r;
  asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(r) : "f"(hi), "f"(lo));
  return r;
}
// eight bf16 (one 16-byte granule) times `scale` -> eight codes (8 bytes, element order)
__device__ __forceinline__ uint2 e4m3x8(uint4 v, float scale) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  uint32_t c[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float lo = __uint_as_float(w[i] << 16) * scale;
    const float hi = __uint_as_float(w[i] & 0xFFFF0000u) * scale;
    c[i] = e4m3x2(lo, hi);
  }
  return make_uint2(c[0] | (c[1] << 16), c[2] | (c[3] << 16));
}
// max |x| of eight bf16 (one granule), exact in fp32
__device__ __forceinline__ float absmax8(uint4 v) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  float m = 0.0f;
#pragma unroll
  for (int i = 0; i < 4; ++i)
    m = fmaxf(m, fmaxf(fabsf(__uint_as_float(w[i] << 16)), fabsf(__uint_as_float(w[i] & 0xFFFF0000u))));
  return m;
}
// Query row exponent: the smallest e with amax <= 448 * 2^e, from the bit fields of amax
// (>= 0).  With amax = 1.f 2^E, i.e. m 2^(E+1) for m = 1.f / 2 in [0.5, 1), and 448 = 0.875 *
// 2^9: e = E - 8 when m <= 0.875 (1.f <= 1.75: mantissa field <= 0x600000), else E - 7.  Zero
// gives 0; subnormal amax (below 2^-126) and anything beyond [-120, 120] is clamped.
__device__ __forceinline__ int e4m3_row_exponent(float amax) {
  const uint32_t b = __float_as_uint(amax);
  if (b == 0) return 0;
  if ((b >> 23) == 0) return -120;
  const int E = (int)(b >> 23) - 127;
  const int e = (b & 0x7FFFFFu) <= 0x600000u ? E - 8 : E - 7;
  return max(-120, min(120, e));
}
// 2^k as a float for k in [-126, 127] (exact)
__device__ __forceinline__ float pow2f(int k) { return __uint_as_float((uint32_t)(127 + k) << 23); }

// Score contract (Eq. 3 under the kernel's precision), shared by the scoring kernel and the
// current-chunk kernel.  Two channels (one 32-bit word: low half first) of the norm and dot fma
// chains, with the bf16 values used directly as fma operands (fp32 product and accumulation, one
// rounding): n += c*c and d += p*c for the low channel, then for the high channel.
__device__ __forceinline__ void fma_word(uint32_t cw, uint32_t pw, float& n, float& d) {
  asm("{\n .reg .b16 cl, ch, pl, ph;\n mov.b32 {cl, ch}, %2;\n mov.b32 {pl, ph}, %3;\n"
      " fma.rn.f32.bf16 %0, cl, cl, %0;\n fma.rn.f32.bf16 %1, pl, cl, %1;\n"
      " fma.rn.f32.bf16 %0, ch, ch, %0;\n fma.rn.f32.bf16 %1, ph, ch, %1;\n}"
      : "+f"(n), "+f"(d) : "r"(cw), "r"(pw));
}

// trunc(v * 2^24) = hi * 2^24 + lo exactly, as two int32: hi = trunc(v) (|hi| <= 2^23 under
// the precondition), v - hi is exact in fp32 (the low-order bits of v), lo = trunc((v - hi) *
// 2^24) with |lo| < 2^24; hi and lo carry the sign of v, so both truncations go toward zero.
// 32-bit conversions only (a float-to-int64 conversion would run on the FP64 pipe).
__device__ __forceinline__ void fixed24_split(float v, int& hi, int& lo) {
  hi = __float2int_rz(v);
  lo = __float2int_rz(__fmul_rn(__fsub_rn(v, __int2float_rn(hi)), 16777216.0f));
}
#endif

// ------------------------------------------------------------------ copy kernels
// Current chunk update in one pass: each 16-byte granule of the previous current chunk (in
// the view fronts) is first copied to its history location, then overwritten by the new
// chunk's granule from the caller's token-major [C*F][H][D] buffer.
// The retired chunk's frames pass through the current-chunk kernel's registers; when the layer
// scores its keys, the same kernel forms their score-contract sums (Sec. 4.3, Eq. 3): the
// squared norms N and the dots D with the previous frame, per (head, frame, segment), added into
// the pending scoring run's int64 sums, so no scoring launch re-reads those frames.
constexpr int kFuseMaxFrames = 15;   // chunks of at most this many frames can be scored in-kernel
struct CurrentArgs {
  const bf16* srcK;             // new chunk, token-major; nullptr = retire only
  const bf16* srcV;
  int rows;                     // C*F
  int heads;
  int head_dim;
  int F, S, W, cap_nonsink;
  int retire;                   // 1: the previous current chunk joins the history
  int nh_old;                   // history frames before the retire
  int static_anchor;            // 1: static views keep the anchor frame (Eq. 2)
  bf16* viewK[kMaxHeads];       // view fronts (current chunk rows)
  bf16* viewV[kMaxHeads];
  bf16* pageK[kMaxHeads];       // page rings (nullptr: head keeps no history pages)
  bf16* pageV[kMaxHeads];
  uint8_t* viewK8[kMaxHeads];   // FP8 attention: E4M3 copies of the K views, same rows (else nullptr)
  uint8_t* viewV8[kMaxHeads];   // FP8 P V: E4M3 copies of the V views (else nullptr)
  unsigned char is_static[kMaxHeads];   // static: sink / anchor slots live in the view
  // in-kernel scoring of the retired chunk (requires retire; every retired frame and the frame
  // before the chunk are non-sink window frames, and C <= kFuseMaxFrames)
  int score;                    // 1: form the sums of the retired frames
  int score_partner_norm;       // 1: also N of the frame before the chunk (run frame score_k0)
  int score_k0;                 // run-relative index of the frame before the chunk; retired
                                // frame r is run frame score_k0 + 1 + r
  int n_seg, seg_len, max_run;
  unsigned long long* sums;     // [target][max_run][n_seg][2]: {N, D}, as the scoring kernel
  int* status;
  short score_target[kMaxHeads];   // sums target of head h, -1: not scored
};
void launch_current(const CurrentArgs& a, cudaStream_t s);

struct ScatterArgs {            // token-major [rows][H][D] -> per-head row-major [rows][D]
  const bf16* srcK;
  const bf16* srcV;
  int rows;
  int heads;
  int head_dim;
  bf16* dstK[kMaxHeads];        // nullptr = skip this head
  bf16* dstV[kMaxHeads];
  uint8_t* dstK8[kMaxHeads];    // FP8 attention view rows: E4M3 copy of dstK (else nullptr)
  uint8_t* dstV8[kMaxHeads];    // FP8 P V view rows: E4M3 copy of dstV (else nullptr)
};
void launch_scatter(const ScatterArgs& a, cudaStream_t s);

// ------------------------------------------------------------------ scoring / selection
struct ScoreItem {              // one (layer, head) whose keys are scored
  const bf16* pagesK;           // page ring [ring_slots][F][D]
  int layer;
  int target;
};

struct SelectTarget {           // one kept set: its layer and the score items feeding it
  int layer;
  int first_item;
  int n_items;
};

struct LayerRun {               // per layer: the run of frames t_first..t_first+n_run-1
  int t_first;
  int n_run;                    // frames whose sums the selection kernel finishes; 0 = none
  int t_fresh;                  // frames >= t_fresh may come from the kernel launched just
                                // before (the chunk it retired): read after its completion
  int n_read;                   // frames t_first.. the scoring kernel reads (the rest of the
                                // run's sums were formed by the current-chunk kernel)
};

// Scoring of new frame pairs (score kernel), then the finish of the scores and BottomK
// selection of every target with a run (select kernel, one CTA per target).
struct ScoreArgs {
  const ScoreItem* items;       // device table
  const SelectTarget* targets;  // device table
  int n_items;
  int F, D, n_seg, seg_len, chunks;
  int S, cap_nonsink, ring_slots;
  int max_run;                  // frames one target's sums can hold
  int max_ctas;                 // persistent grid size
  long long total_units;        // frame-chunks of this launch (item, segment, chunk, frame)
  int n_active;                 // layers with a run, ascending
  int act_layer[kMaxLayers];
  int act_first_item[kMaxLayers];   // first score item of the layer
  long long act_start[kMaxLayers];  // first frame-chunk of the layer in the flattened range
  int scope;                    // FK_SCOPE_*
  int rule;                     // FK_SELECT_*: similarity scores, or a comparison rule's values
  unsigned int seed;            // FK_SELECT_RANDOM
  int k_frame;                  // kept per frame (per-frame scope)
  int kmax;                     // capacity of one kept list
  unsigned long long* sums;     // scratch [target][max_run][n_seg][2] : {N(t), D(t-1,t)}, zero between launches
  float* scores;                // [target][ring_slots][n_seg]
  int* kept;                    // [target][kmax]
  int* status;
  LayerRun run[kMaxLayers];
  int t_lo[kMaxLayers];         // first scoreable frame of the window
  int n_scoreable[kMaxLayers];  // |T| (scoreable frames)
  int n_keep[kMaxLayers];       // kept segments of the layer's targets
};
void launch_score(const ScoreArgs& a, cudaStream_t s);
void launch_select(const ScoreArgs& a, int n_targets, cudaStream_t s);
// one-thread kernel whose bounded wait expires after limit_ns (failure-detection self-test)
cudaError_t launch_wait_selftest(uint64_t limit_ns, int* status, cudaStream_t s);
// dynamic shared memory limits and the persistent grid size (CTAs resident at once)
cudaError_t score_prepare(int head_dim, int max_run, int n_seg, int* max_ctas);
// frame-chunks in flight per scoring CTA (one bulk copy each)
constexpr int kScoreStages = 6;
constexpr int kSelectThreads = 256;

struct CompactItem {            // one dynamic (layer, head)
  const bf16* pagesK;
  const bf16* pagesV;
  bf16* viewK;
  bf16* viewV;
  int layer;
  int target;                   // kept list
  uint8_t* viewK8;              // FP8 attention: E4M3 copy of the K view, same rows (else nullptr)
  uint8_t* viewV8;              // FP8 P V: E4M3 copy of the V view (else nullptr)
};

struct CompactArgs {
  const CompactItem* items;
  int n_items;
  int F, D, n_seg, seg_len, CF;
  int S, cap_nonsink, kmax;
  int splits;                   // pieces per unit (each at most kCompactPiece bytes per tensor)
  int units_per_cta;            // whole units per CTA when a unit is smaller (then splits = 1)
  const int* kept;
  // per layer: the kept segments this launch copies into the dynamic views' kept-segment rings
  // (views are [current | sinks | anchor | kept ring of kmax segment slots]; the sinks and the
  // anchor are written by the current-chunk and prefill kernels)
  int n_kept_copy[kMaxLayers];  // kept segments to copy
  int kp0[kMaxLayers];          // their first position in the target's kept list
  int rp0[kMaxLayers];          // ring slot of the first one (slots wrap modulo kmax)
  unsigned char active[kMaxLayers];
  int max_units;
};
constexpr int kCompactPiece = 16384;
void launch_compact(const CompactArgs& a, cudaStream_t s);
// streaming read of `bytes` (a multiple of 16) from 16-byte aligned device memory: calibration
cudaError_t launch_stream_read(const void* src, int64_t bytes, cudaStream_t s);

// ------------------------------------------------------------------ attention
struct AttnArgs {
  bf16* O;                      // [Nq][H][D]
  int Nq;
  int H;
  int n_qtiles;
  float scale_log2;             // log2(e) / sqrt(D)
  int* status;
  int kv_splits;                // key splits per (head, query-tile pair): 1, or 2 with a merge
  float* part_o;                // [kv_splits][Nq][H][D] unnormalised split outputs (kv_splits > 1)
  float2* part_ml;              // [kv_splits][Nq][H] {running max (log2 domain), row sum}
  int head_of[kMaxHeads];       // CTA order: head index of the i-th (longest-first) head
  int row_base[kMaxHeads];      // first row of the head's packed view in the view arena
  int n_keys[kMaxHeads];        // keys the head attends to
};
// tmQ: 3D map over Q [Nq][H][D]; tmK/tmV: 2D maps over the view arenas [rows][D].
// precision FK_ATTN_FP8_QK: Q K^T on E4M3 operands (head_dim 128): tmK then maps the E4M3 key
// arena (box 128 x 128, one 128-byte swizzle atom per row); tmQ still maps the bf16 queries,
// which the kernel quantizes itself.  FK_ATTN_FP8: P V on E4M3 operands too: tmV maps the
// E4M3 value arena the same way.
void launch_attention(int head_dim, int precision, const CUtensorMap& tmQ, const CUtensorMap& tmK,
                      const CUtensorMap& tmV, const AttnArgs& a, cudaStream_t s);
cudaError_t attention_prepare(int head_dim);   // sets the dynamic shared-memory limits
// combine the key splits of every (row, head) into O (bf16)
void launch_merge(int head_dim, const AttnArgs& a, cudaStream_t s);
constexpr int kMaxKvSplits = 2;

// ------------------------------------------------------------------ FP8 (E4M3) quantization
// One launch: the query rows (part 0, row-scaled) and key row ranges of a [rows][k_dim] bf16
// arena (parts 1..n, unscaled) into byte arrays of the same shapes.
struct QuantArgs {
  const bf16* q_src;            // [q_rows][q_dim] bf16 (q_rows = 0: no query part)
  uint8_t* q_dst;               // [q_rows][q_dim] E4M3 codes
  int8_t* q_exp;                // [q_rows] row exponents
  int64_t q_rows;
  int q_dim;                    // 64 or 128
  const bf16* k_src;            // key arena [rows][k_dim] bf16
  uint8_t* k_dst;               // its E4M3 copy [rows][k_dim]
  int k_dim;                    // a multiple of 8
  int n;                        // key ranges, <= kMaxHeads
  int64_t row0[kMaxHeads];      // range i: rows [row0[i], row0[i] + rows[i])
  int64_t rows[kMaxHeads];
  int64_t blk[kMaxHeads + 2];   // first block of each part, set by launch_quant
};
void launch_quant(QuantArgs& a, cudaStream_t s);

// ------------------------------------------------------------------ head profiling (Eq. 1)
struct ProfArgs {
  int Nq, Nk, H, n_qtiles;
  float scale_log2;             // log2(e) / sqrt(D)
  int g_end;                    // keys [0, g_end): generated chunk
  int s_end;                    // keys [g_end, s_end): sink frames
  int t_begin;                  // keys [t_begin, Nk): transition frame; the rest: other history
  double* mass;                 // [H][4]: rows, generated, transition, sink (added to)
  int* status;
};
// tmQ / tmK: 3D maps over Q [Nq][H][D] and K [Nk][H][D] (128-row boxes, 128-byte swizzle)
cudaError_t launch_head_profile(int head_dim, const CUtensorMap& tmQ, const CUtensorMap& tmK,
                                const ProfArgs& a, cudaStream_t s);

}  // namespace fk
