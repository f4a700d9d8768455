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
constexpr int kScoreTokens = 32;      // tokens of one segment handled by one scoring CTA

// device status word bits (set by kernels, read by fk_sync_status)
constexpr int kStatusRange = 1;
constexpr int kStatusTimeout = 2;

// ------------------------------------------------------------------ copy kernels
struct ScatterArgs {            // token-major [rows][H][D] -> per-head row-major [rows][D]
  const bf16* srcK;
  const bf16* srcV;
  int rows;
  int heads;
  int head_dim;
  bf16* dstK[kMaxHeads];        // nullptr = skip this head
  bf16* dstV[kMaxHeads];
};

struct CopyJob {                // contiguous byte copy, 16-byte granules
  const void* src;
  void* dst;
  int64_t bytes;
};
constexpr int kMaxCopyJobs = 512;
struct CopyJobs {
  int n;
  CopyJob job[kMaxCopyJobs];
};

void launch_scatter(const ScatterArgs& a, cudaStream_t s);
void launch_copy_jobs(const CopyJobs& j, cudaStream_t s);

// ------------------------------------------------------------------ scoring / selection
struct ScoreItem {              // one (layer, head) whose keys are scored
  const bf16* pagesK;           // page ring [ring_slots][F][D]
  int layer;
  int target;
};

struct LayerRun {               // per layer: frames t_first..t_first+n_run-1 are read
  int t_first;
  int n_run;                    // 0 = nothing to score in this layer
};

struct ScoreArgs {
  const ScoreItem* items;       // device table
  int n_items;
  int F, D, n_seg, seg_len, chunks;
  int S, cap_nonsink;
  int max_run;
  long long* partials;          // [item][max_run][n_seg][chunks][2] : {N, Dnext}
  int* status;
  LayerRun run[kMaxLayers];
};
void launch_score(const ScoreArgs& a, cudaStream_t s);

struct SelectTarget {           // per target (selection unit)
  int layer;                    // layer whose frames the target covers
  int first_item;               // score items feeding the target: [first_item, first_item+n_items)
  int n_items;
};

struct SelectArgs {
  const SelectTarget* targets;  // device table
  int n_targets;
  int n_seg, chunks, max_run;
  int S, cap_nonsink, ring_slots;
  int scope;                    // FK_SCOPE_*
  int k_frame;                  // kept per frame (per-frame scope)
  int kmax;                     // capacity of one kept list
  const long long* partials;
  float* scores;                // [target][ring_slots][n_seg]
  int* kept;                    // [target][kmax]
  LayerRun run[kMaxLayers];     // frames scored now (as in ScoreArgs)
  int t_lo[kMaxLayers];         // first scoreable frame of the window
  int n_scoreable[kMaxLayers];  // |T| (scoreable frames)
  int n_keep[kMaxLayers];       // kept segments of the layer's targets
};
void launch_select(const SelectArgs& a, cudaStream_t s);

struct CompactItem {            // one dynamic (layer, head)
  const bf16* pagesK;
  const bf16* pagesV;
  bf16* viewK;
  bf16* viewV;
  int layer;
  int target;                   // kept list
};

struct CompactArgs {
  const CompactItem* items;
  int n_items;
  int F, D, n_seg, seg_len, CF;
  int S, cap_nonsink, kmax;
  const int* kept;
  int n_sink_present[kMaxLayers];
  int n_keep[kMaxLayers];
  int anchor[kMaxLayers];       // -1 = none
  unsigned char active[kMaxLayers];
  int max_units;
};
void launch_compact(const CompactArgs& a, cudaStream_t s);

// ------------------------------------------------------------------ attention
struct AttnArgs {
  bf16* O;                      // [Nq][H][D]
  int Nq;
  int H;
  int n_qtiles;
  float scale_log2;             // log2(e) / sqrt(D)
  int* status;
  int head_of[kMaxHeads];       // CTA order: head index of the i-th (longest-first) head
  int row_base[kMaxHeads];      // first row of the head's packed view in the view arena
  int n_keys[kMaxHeads];        // keys the head attends to
};
// tmQ: 3D map over Q [Nq][H][D]; tmK/tmV: 2D maps over the view arenas [rows][D].
void launch_attention(int head_dim, const CUtensorMap& tmQ, const CUtensorMap& tmK,
                      const CUtensorMap& tmV, const AttnArgs& a, cudaStream_t s);
cudaError_t attention_prepare(int head_dim);   // sets the dynamic shared-memory limit

}  // namespace fk
