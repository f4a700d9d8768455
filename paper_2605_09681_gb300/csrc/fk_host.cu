// Host side of the Forcing-KV library: configuration checks, device-memory layout,
// frame bookkeeping (sink / window / anchor / scoreable frames, Sec. 4.2-4.3, App. H)
// and the C ABI declared in fk.h.  All arithmetic of the method runs in the kernels
// of fk_copy.cu, fk_score.cu and fk_attn.cu; this file only decides what to launch.
//
// Device memory (allocated once in fk_create, zero-initialised):
//   view arenas  K and V, [rows][D] bf16 each; head (l, h) owns rows
//                [row_base, row_base + view_rows), padded to whole 128-key tiles.
//                Static head view:  [current chunk C*F | sink S*F | anchor F]
//                Dynamic head view: [current chunk C*F | sink S*F | anchor F | kept-segment
//                ring of kmax slots] (attention does not depend on the key order)
//   page rings   K and V, [ring_slots][F][D] per head that keeps history for scoring
//                (dynamic heads; every head of layer 0 under layer-0 pooled scoring);
//                frame f lives in slot f (f < S) or S + (f - S) mod cap_nonsink.
//   scores       fp32 [target][ring_slots][n]; kept lists int32 [target][kmax];
//                int64 scoring sums (scratch); status word;
//                host staging (two slots of K, V and Q; O) and the attention key-split
//                scratch (fp32 partial outputs and row statistics of two splits).
//   FP8 only     the E4M3 copy of the K view arena ([rows][D] bytes, written by the copy
//                kernels together with every bf16 view K row) and, when P V also runs on
//                E4M3 (FK_ATTN_FP8), of the V view arena; the attention kernel quantizes
//                its query tiles itself.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <new>
#include <queue>
#include <vector>

#include <cudaTypedefs.h>

#include "fk_internal.h"

using namespace fk;

namespace {

struct HeadBuf {
  bool is_static = false;
  bool retains = false;   // owns a page ring
  bf16* pageK = nullptr;
  bf16* pageV = nullptr;
  bf16* viewK = nullptr;
  bf16* viewV = nullptr;
  int64_t row_base = 0;
  int view_rows = 0;
  int target = -1;        // selection target (dynamic heads)
};

struct LayerState {
  int nh = 0;             // history frames appended
  bool has_current = false;
  bool dirty = false;     // appended since the last fk_compress
  int scored_upto = 0;    // pairs (t, t+1) with t < scored_upto are scored
  int n_keep = 0;         // kept segments of each dynamic head (after fk_compress)
  int len_static = 0;     // keys of a static head
  int len_dynamic = 0;    // keys of a dynamic head
  // incremental compaction: the dynamic views' kept-segment ring holds the kept segments of
  // frames [ring_first, ring_end), the first of them at ring slot ring_head
  int ring_first = 0;
  int ring_end = 0;
  int ring_head = 0;
  // scoring sums formed by the current-chunk kernel since the last fk_compress: 0 none,
  // 1 the sums of run frames [fuse_t_first, fuse_end) except the first fuse_n_read (which the
  // scoring kernel reads), 2 sums that match no run (fk_compress clears them and rescores)
  int fuse_state = 0;
  int fuse_t_first = 0;
  int fuse_end = 0;
  int fuse_n_read = 0;
};

struct Staging {
  bf16* buf[2][2] = {};           // [slot][tensor]
  cudaEvent_t ready[2] = {}, freed[2] = {};
  int slot = 0;                   // next slot to fill
};

struct ProfRec {
  int kind;
  cudaEvent_t a, b;
};

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_encode_once;

bool get_encode() {
  std::call_once(g_encode_once, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  });
  return g_encode != nullptr;
}

int64_t round_up(int64_t x, int64_t m) { return (x + m - 1) / m * m; }

// Key splits of one attention launch.  The CTAs (one per SM) are dispatched longest first;
// the makespan on n_sms SMs is estimated greedily in units of key tiles (plus a fixed cost
// per CTA), without and with 2 key splits (plus the merge pass); equal-length heads whose CTAs
// fill 1.5 waves are where the split pays.
int choose_kv_splits(int n_sms, int n_qtiles, int CF, int H, int D, const int* n_keys) {
  const double kOverheadTiles = 3.0, kTileUs = 1.65, kHbmBytesPerUs = 6.0e6;
  auto makespan = [&](int sp) {
    std::vector<double> d;
    for (int hd = 0; hd < H; ++hd) {
      const int nt = (n_keys[hd] + kAttnBN - 1) / kAttnBN;
      if (nt < sp) return 1e30;
      for (int q = 0; q < n_qtiles; ++q)
        for (int k = 0; k < sp; ++k) d.push_back((double)((k + 1) * nt / sp - k * nt / sp) + kOverheadTiles);
    }
    std::sort(d.begin(), d.end(), std::greater<double>());
    std::priority_queue<double, std::vector<double>, std::greater<double>> load;
    for (int i = 0; i < n_sms; ++i) load.push(0.0);
    double span = 0.0;
    for (double x : d) {
      const double t = load.top() + x;
      load.pop();
      load.push(t);
      span = std::max(span, t);
    }
    return span;
  };
  const double merge_tiles =
      ((double)kMaxKvSplits * CF * H * D * 4 + (double)CF * H * D * 2) / kHbmBytesPerUs / kTileUs;
  return makespan(2) + merge_tiles < 0.95 * makespan(1) ? 2 : 1;
}

}  // namespace

struct fk_handle {
  fk_config cfg{};
  std::vector<uint8_t> static_map;
  int L = 0, H = 0, D = 0, F = 0, C = 0, S = 0, W = 0, n = 0, b = 0;
  int scope = 0, source = 0, incremental = 0, max_hist = 0, dev = 0;
  int seg = 0, CF = 0;
  int cap_nonsink = 0, ring_slots = 0, k_frame = 0, kmax = 0, chunks = 0;
  int selection = FK_SELECT_SIMILARITY;
  uint32_t select_seed = 0;
  bool drop_anchor = false;        // static heads keep sink + current chunk only
  bool fp8 = false;                // FK_ATTN_FP8_QK or FK_ATTN_FP8: Q K^T on E4M3
  bool fp8pv = false;              // FK_ATTN_FP8: P V on E4M3 too
  int precision = FK_ATTN_BF16;
  std::vector<HeadBuf> heads;      // [L*H]
  std::vector<LayerState> layers;  // [L]
  // device memory
  std::vector<void*> allocs;
  size_t reserved = 0;
  bf16* viewK = nullptr;
  bf16* viewV = nullptr;
  int64_t view_rows_total = 0;
  float* scores = nullptr;
  int* kept = nullptr;
  unsigned long long* sums = nullptr;
  size_t sums_bytes = 0;
  int* status = nullptr;
  // host-input staging: two slots per kind (K with V; Q), each with a ready event (copy done)
  // and a freed event (the kernel that read the slot has run); optional copy stream
  Staging st_kv, st_q;
  // output staging: two slots; with host overlap on, copied back on copy_out_stream
  bf16* stage_o[2] = {};
  cudaEvent_t o_ready[2] = {}, o_copied[2] = {};
  int o_slot = 0;
  bool o_pending[2] = {};
  cudaStream_t copy_out_stream = nullptr;
  int64_t stage_frames = 0;        // frames one K/V staging buffer holds
  cudaStream_t copy_stream = nullptr;
  bool host_overlap = false;
  // attention key splits: scratch for split outputs, SM count, last decision per layer
  float* part_o = nullptr;
  float2* part_ml = nullptr;
  int n_sms = 0;
  std::vector<std::vector<int>> split_keys;   // [L]: key counts the cached decision was made for
  std::vector<int> split_choice;              // [L]
  ScoreItem* d_score_items = nullptr;
  SelectTarget* d_targets = nullptr;
  CompactItem* d_compact_items = nullptr;
  std::vector<ScoreItem> score_items;
  std::vector<std::pair<int, int>> layer_items;   // [L]: first score item, item count
  std::vector<SelectTarget> targets;
  std::vector<int> target_layer;
  std::vector<CompactItem> compact_items;
  int max_run = 0;
  int score_ctas = 0;
  CUtensorMap tmK{}, tmV{};
  uint8_t* viewK8 = nullptr;       // FP8: E4M3 codes of the K view arena
  CUtensorMap tmK8{};
  uint8_t* viewV8 = nullptr;       // FP8 P V: E4M3 codes of the V view arena
  CUtensorMap tmV8{};
  const void* q_cached[2] = {};   // two cached Q maps (the two Q staging slots alternate)
  CUtensorMap tmQ[2]{};
  int q_next = 0;
  // profiling
  bool prof = false;
  std::vector<ProfRec> prof_pending;
  std::vector<cudaEvent_t> ev_free;
  double prof_ms[FK_KERNEL_KINDS] = {};
  int64_t prof_n[FK_KERNEL_KINDS] = {};
  int64_t launches = 0;
};

namespace {

fk_status cuda_fail(cudaError_t e) {
  return e == cudaErrorMemoryAllocation ? FK_ERR_NOMEM : FK_ERR_CUDA;
}

#define FK_CUDA(x)                                  \
  do {                                              \
    cudaError_t e_ = (x);                           \
    if (e_ != cudaSuccess) return cuda_fail(e_);    \
  } while (0)

bool is_device_ptr(const void* p) {
  cudaPointerAttributes at{};
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int ring_slot(const fk_handle* h, int f) {
  return f < h->S ? f : h->S + (f - h->S) % h->cap_nonsink;
}

struct Roles {
  int n_sink;       // sink frames present
  int lo;           // first window frame
  int anchor;       // -1 = none
  int t_lo;         // first scoreable frame
  int n_scoreable;  // scoreable frames t_lo .. t_lo + n - 1
};

Roles roles_of(const fk_handle* h, int nh) {
  Roles r{};
  r.n_sink = std::min(h->S, nh);
  r.lo = h->W > 0 ? std::max(h->S, nh - h->W) : h->S;
  r.anchor = nh - 1 >= r.lo ? nh - 1 : -1;
  r.t_lo = r.lo;
  r.n_scoreable = r.anchor >= 0 ? r.anchor - r.lo : 0;
  return r;
}

int keep_total(const fk_handle* h, int n_scoreable) {
  if (h->scope == FK_SCOPE_PER_FRAME) return n_scoreable * h->k_frame;
  if (h->selection == FK_SELECT_ALL) return n_scoreable * h->n;
  return (int)(((int64_t)h->b * n_scoreable * h->n) / 1000);
}

void update_lengths(fk_handle* h, int l) {
  LayerState& ls = h->layers[l];
  const Roles r = roles_of(h, ls.nh);
  const int base = h->CF + r.n_sink * h->F;
  const int anchor_rows = r.anchor >= 0 ? h->F : 0;
  ls.len_static = base + (h->drop_anchor ? 0 : anchor_rows);
  ls.len_dynamic = base + anchor_rows + ls.n_keep * h->seg;
}

// ---- profiling and launch accounting
void prof_begin(fk_handle* h, cudaStream_t s, cudaEvent_t* ev) {
  *ev = nullptr;
  if (!h->prof || h->ev_free.size() < 2) return;
  *ev = h->ev_free.back();
  h->ev_free.pop_back();
  cudaEventRecord(*ev, s);
}

void prof_end(fk_handle* h, cudaStream_t s, int kind, cudaEvent_t ev0) {
  h->launches++;
  if (!ev0) return;
  cudaEvent_t ev1 = h->ev_free.back();
  h->ev_free.pop_back();
  cudaEventRecord(ev1, s);
  h->prof_pending.push_back({kind, ev0, ev1});
}

fk_status prof_collect(fk_handle* h) {
  for (auto& r : h->prof_pending) {
    FK_CUDA(cudaEventSynchronize(r.b));
    float ms = 0.f;
    FK_CUDA(cudaEventElapsedTime(&ms, r.a, r.b));
    h->prof_ms[r.kind] += ms;
    h->prof_n[r.kind] += 1;
    h->ev_free.push_back(r.a);
    h->ev_free.push_back(r.b);
  }
  h->prof_pending.clear();
  return FK_OK;
}

template <class F>
fk_status launch(fk_handle* h, cudaStream_t s, int kind, F&& f) {
  cudaEvent_t ev0;
  if (h->prof && h->ev_free.size() < 4) prof_collect(h);
  prof_begin(h, s, &ev0);
  f();
  cudaError_t e = cudaGetLastError();
  prof_end(h, s, kind, ev0);
  return e == cudaSuccess ? FK_OK : FK_ERR_CUDA;
}

fk_status dev_alloc(fk_handle* h, size_t bytes, void** out) {
  *out = nullptr;
  if (bytes == 0) return FK_OK;
  void* p = nullptr;
  cudaError_t e = cudaMalloc(&p, bytes);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return cuda_fail(e);
  }
  h->allocs.push_back(p);
  h->reserved += bytes;
  e = cudaMemset(p, 0, bytes);
  if (e != cudaSuccess) return FK_ERR_CUDA;
  *out = p;
  return FK_OK;
}

// Host inputs [rows][H][D] (up to two of `bytes` each) into the next staging slot of `sg`;
// device inputs pass through.  *slot is the slot used, -1 when nothing was staged; the caller
// records sg.freed[*slot] on `s` after the kernel that reads it.  By default the copies run on
// `s` in call order; with host overlap on, they run at once on the copy stream (after the
// slot's previous reader) and `s` waits for them before the reader.
fk_status stage_inputs(fk_handle* h, Staging& sg, const void* a, const void* b, size_t bytes,
                       cudaStream_t s, const bf16** oa, const bf16** ob, int* slot) {
  const void* src[2] = {a, b};
  const bf16** out[2] = {oa, ob};
  bool host[2] = {false, false};
  for (int i = 0; i < 2; ++i) {
    if (!src[i]) continue;
    host[i] = !is_device_ptr(src[i]);
    if (!host[i]) *out[i] = static_cast<const bf16*>(src[i]);
  }
  *slot = -1;
  if (!host[0] && !host[1]) return FK_OK;
  const int sl = sg.slot;
  sg.slot ^= 1;
  cudaStream_t cs = h->host_overlap ? h->copy_stream : s;
  if (h->host_overlap) FK_CUDA(cudaStreamWaitEvent(cs, sg.freed[sl], 0));
  for (int i = 0; i < 2; ++i) {
    if (!host[i]) continue;
    FK_CUDA(cudaMemcpyAsync(sg.buf[sl][i], src[i], bytes, cudaMemcpyHostToDevice, cs));
    *out[i] = sg.buf[sl][i];
  }
  if (h->host_overlap) {
    FK_CUDA(cudaEventRecord(sg.ready[sl], cs));
    FK_CUDA(cudaStreamWaitEvent(s, sg.ready[sl], 0));
  }
  *slot = sl;
  return FK_OK;
}

// 2D map over a [rows][D] arena, 128-row boxes of one 128-byte swizzle atom per row: 64 bf16
// (bf16) or 128 E4M3 codes (e4m3, D = 128)
fk_status encode_2d(CUtensorMap* m, void* base, int64_t rows, int D, bool e4m3 = false) {
  const cuuint64_t dims[2] = {(cuuint64_t)D, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)D * (e4m3 ? 1 : 2)};
  const cuuint32_t box[2] = {e4m3 ? 128u : 64u, (cuuint32_t)kAttnBN};
  const cuuint32_t es[2] = {1, 1};
  CUresult r = g_encode(m, e4m3 ? CU_TENSOR_MAP_DATA_TYPE_UINT8 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16,
                        2, base, dims, strides, box, es,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? FK_OK : FK_ERR_CUDA;
}

fk_status encode_q(CUtensorMap* m, const void* q, int Nq, int H, int D) {
  const cuuint64_t dims[3] = {(cuuint64_t)D, (cuuint64_t)H, (cuuint64_t)Nq};
  const cuuint64_t strides[2] = {(cuuint64_t)D * 2, (cuuint64_t)H * D * 2};
  const cuuint32_t box[3] = {64, 1, (cuuint32_t)kAttnBM};
  const cuuint32_t es[3] = {1, 1, 1};
  CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(q), dims,
                        strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? FK_OK : FK_ERR_CUDA;
}

// Prefill: append nf frames from token-major [nf*F][H][D] device buffers to the history.
fk_status push_history(fk_handle* h, int layer, const bf16* tokK, const bf16* tokV, int nf,
                       cudaStream_t s) {
  LayerState& ls = h->layers[layer];
  const int nh0 = ls.nh, nh1 = ls.nh + nf;
  const int lo1 = h->W > 0 ? std::max(h->S, nh1 - h->W) : h->S;   // window after the push
  const int64_t frame_elems = (int64_t)h->F * h->D;
  for (int i = 0; i < nf; ++i) {
    const int f = nh0 + i;
    const bool sink = f < h->S;
    const bool in_window = sink || f >= lo1;        // frames overwritten within this push are skipped
    const bool is_anchor = !sink && f == nh1 - 1;
    if (!in_window) continue;
    ScatterArgs pa{}, va{};
    pa.srcK = tokK + (int64_t)i * h->F * h->H * h->D;
    pa.srcV = tokV + (int64_t)i * h->F * h->H * h->D;
    pa.rows = h->F;
    pa.heads = h->H;
    pa.head_dim = h->D;
    va = pa;
    bool any_p = false, any_v = false;
    for (int hd = 0; hd < h->H; ++hd) {
      const HeadBuf& hb = h->heads[layer * h->H + hd];
      if (hb.retains) {
        pa.dstK[hd] = hb.pageK + ring_slot(h, f) * frame_elems;
        pa.dstV[hd] = hb.pageV + ring_slot(h, f) * frame_elems;
        any_p = true;
      }
      // every view holds the sinks; every dynamic view (and, unless they drop it, every
      // static view) holds the anchor
      if (sink || (is_anchor && (!hb.is_static || !h->drop_anchor))) {
        const int64_t row = h->CF + (int64_t)(sink ? f : h->S) * h->F;
        va.dstK[hd] = hb.viewK + row * h->D;
        va.dstV[hd] = hb.viewV + row * h->D;
        if (h->fp8) va.dstK8[hd] = h->viewK8 + (hb.row_base + row) * h->D;
        if (h->fp8pv) va.dstV8[hd] = h->viewV8 + (hb.row_base + row) * h->D;
        any_v = true;
      }
    }
    if (any_p) {
      fk_status st = launch(h, s, FK_KERNEL_APPEND, [&] { launch_scatter(pa, s); });
      if (st != FK_OK) return st;
    }
    if (any_v) {
      fk_status st = launch(h, s, FK_KERNEL_APPEND, [&] { launch_scatter(va, s); });
      if (st != FK_OK) return st;
    }
  }
  ls.nh = nh1;
  ls.dirty = true;
  if (ls.fuse_state == 1) ls.fuse_state = 2;   // frames the fused sums do not cover
  update_lengths(h, layer);
  return FK_OK;
}

// Whether the current-chunk kernel that retires layer `layer`'s current chunk can form the
// pending scoring run's sums of the retired frames itself (Eq. 3 under the score contract):
// the layer scores keys, the chunk has at most kFuseMaxFrames frames, the frame before the
// chunk is a non-sink frame that stays in the window, and no other append since the last
// fk_compress has touched the sums.  Fills the kernel's scoring fields and the layer's state.
void plan_fused_scoring(fk_handle* h, int layer, CurrentArgs& a) {
  LayerState& ls = h->layers[layer];
  if (h->selection != FK_SELECT_SIMILARITY || h->layer_items[layer].second == 0) return;
  const int anchor_old = ls.nh - 1, nh_new = ls.nh + h->C;
  const int lo_new = h->W > 0 ? std::max(h->S, nh_new - h->W) : h->S;
  bool ok = ls.fuse_state == 0 && h->C <= kFuseMaxFrames && anchor_old >= h->S && anchor_old >= lo_new;
  int t_first = lo_new;            // whole-window rescoring: the run starts at the window
  if (ok && h->incremental) {      // incremental: the run starts at the last scored anchor
    ok = ls.scored_upto == anchor_old;
    t_first = anchor_old;
  }
  if (!ok) {
    if (ls.fuse_state == 1) ls.fuse_state = 2;
    return;
  }
  a.score = 1;
  a.score_partner_norm = h->incremental ? 1 : 0;
  a.score_k0 = anchor_old - t_first;
  a.n_seg = h->n;
  a.seg_len = h->seg;
  a.max_run = h->max_run;
  a.sums = h->sums;
  a.status = h->status;
  const bool pooled = h->source == FK_SCORE_LAYER0_POOLED;
  for (int hd = 0; hd < h->H; ++hd) {
    const HeadBuf& hb = h->heads[layer * h->H + hd];
    a.score_target[hd] = (short)(pooled ? 0 : (hb.is_static ? -1 : hb.target));
  }
  ls.fuse_state = 1;
  ls.fuse_t_first = t_first;
  ls.fuse_end = nh_new;
  // the scoring kernel reads frames t_first .. anchor_old unless the kernel forms N(anchor_old)
  ls.fuse_n_read = a.score_partner_norm ? 0 : a.score_k0 + 1;
}

// One pass of the current-chunk kernel: optionally retire the current chunk (view fronts)
// into the history, optionally write a new current chunk from K/V (host or device).
fk_status update_current(fk_handle* h, int layer, bool retire, const void* K, const void* V,
                         cudaStream_t s) {
  LayerState& ls = h->layers[layer];
  retire = retire && ls.has_current;
  if (retire && h->W == 0 && ls.nh + h->C > h->max_hist) return FK_ERR_FULL;
  const bf16 *k = nullptr, *v = nullptr;
  int slot = -1;
  if (K) {
    const size_t bytes = (size_t)h->CF * h->H * h->D * 2;
    fk_status st = stage_inputs(h, h->st_kv, K, V, bytes, s, &k, &v, &slot);
    if (st != FK_OK) return st;
  }
  if (!retire && !k) return FK_OK;
  CurrentArgs a{};
  a.srcK = k;
  a.srcV = v;
  a.rows = h->CF;
  a.heads = h->H;
  a.head_dim = h->D;
  a.F = h->F;
  a.S = h->S;
  a.W = h->W;
  a.cap_nonsink = h->cap_nonsink;
  a.retire = retire ? 1 : 0;
  a.static_anchor = h->drop_anchor ? 0 : 1;
  a.nh_old = ls.nh;
  for (int hd = 0; hd < h->H; ++hd) {
    const HeadBuf& hb = h->heads[layer * h->H + hd];
    a.viewK[hd] = hb.viewK;
    a.viewV[hd] = hb.viewV;
    a.pageK[hd] = hb.retains ? hb.pageK : nullptr;
    a.pageV[hd] = hb.retains ? hb.pageV : nullptr;
    a.viewK8[hd] = h->fp8 ? h->viewK8 + hb.row_base * h->D : nullptr;
    a.viewV8[hd] = h->fp8pv ? h->viewV8 + hb.row_base * h->D : nullptr;
    a.is_static[hd] = hb.is_static ? 1 : 0;
  }
  if (retire) plan_fused_scoring(h, layer, a);
  fk_status st = launch(h, s, FK_KERNEL_APPEND, [&] { launch_current(a, s); });
  if (st != FK_OK) return st;
  if (slot >= 0) FK_CUDA(cudaEventRecord(h->st_kv.freed[slot], s));
  if (retire) {
    ls.nh += h->C;
    ls.dirty = true;
  }
  ls.has_current = k != nullptr || (ls.has_current && !retire);
  update_lengths(h, layer);
  return FK_OK;
}

}  // namespace

extern "C" {

fk_status fk_head_profile(const void* Q, const void* K, int n_queries, int n_keys, int n_heads,
                          int head_dim, int n_generate, int n_sink, int n_transition, double* mass,
                          int* status, void* stream) {
  if (!Q || !K || !mass || !status) return FK_ERR_ARG;
  if (!aligned16(Q) || !aligned16(K) || (reinterpret_cast<uintptr_t>(mass) & 7u) ||
      (reinterpret_cast<uintptr_t>(status) & 3u))
    return FK_ERR_ARG;
  if (head_dim != 64 && head_dim != 128) return FK_ERR_CONFIG;
  if (n_heads < 1 || n_heads > kMaxHeads || n_queries < 1 || n_keys < 1) return FK_ERR_CONFIG;
  if (n_generate < 0 || n_sink < 0 || n_transition < 0 ||
      (int64_t)n_generate + n_sink + n_transition > n_keys)
    return FK_ERR_CONFIG;
  const int64_t n_qtiles = (n_queries + kAttnBM - 1) / kAttnBM;
  if (2 * n_qtiles * n_heads >= ((int64_t)1 << 31)) return FK_ERR_CONFIG;
  if (!is_device_ptr(Q) || !is_device_ptr(K) || !is_device_ptr(mass) || !is_device_ptr(status))
    return FK_ERR_ARG;
  if (!get_encode()) return FK_ERR_CUDA;
  CUtensorMap tq{}, tk{};
  fk_status st;
  if ((st = encode_q(&tq, Q, n_queries, n_heads, head_dim)) != FK_OK) return st;
  if ((st = encode_q(&tk, K, n_keys, n_heads, head_dim)) != FK_OK) return st;
  ProfArgs a{};
  a.Nq = n_queries;
  a.Nk = n_keys;
  a.H = n_heads;
  a.n_qtiles = (int)n_qtiles;
  a.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)head_dim));
  a.g_end = n_generate;
  a.s_end = n_generate + n_sink;
  a.t_begin = n_keys - n_transition;
  a.mass = mass;
  a.status = status;
  return launch_head_profile(head_dim, tq, tk, a, static_cast<cudaStream_t>(stream)) == cudaSuccess
             ? FK_OK
             : FK_ERR_CUDA;
}

fk_status fk_quantize_e4m3(const void* X, int64_t rows, int dim, int row_scaled, void* q8,
                           int8_t* exps, void* stream) {
  if (!X || !q8 || !aligned16(X) || !aligned16(q8)) return FK_ERR_ARG;
  if (row_scaled != 0 && row_scaled != 1) return FK_ERR_CONFIG;
  if (rows < 0 || rows > ((int64_t)1 << 31)) return FK_ERR_CONFIG;
  if (row_scaled ? (dim != 64 && dim != 128) : (dim < 8 || dim > 1024 || dim % 8)) return FK_ERR_CONFIG;
  if (row_scaled && !exps) return FK_ERR_ARG;
  if (rows == 0) return FK_OK;
  if (!is_device_ptr(X) || !is_device_ptr(q8) || (row_scaled && !is_device_ptr(exps))) return FK_ERR_ARG;
  QuantArgs qa{};
  if (row_scaled) {
    qa.q_src = static_cast<const bf16*>(X);
    qa.q_dst = static_cast<uint8_t*>(q8);
    qa.q_exp = exps;
    qa.q_rows = rows;
    qa.q_dim = dim;
  } else {
    qa.k_src = static_cast<const bf16*>(X);
    qa.k_dst = static_cast<uint8_t*>(q8);
    qa.k_dim = dim;
    qa.n = 1;
    qa.rows[0] = rows;
  }
  launch_quant(qa, static_cast<cudaStream_t>(stream));
  return cudaGetLastError() == cudaSuccess ? FK_OK : FK_ERR_CUDA;
}

fk_status fk_classify_heads(const double* mass, int n_heads, int alpha_permille,
                            uint8_t* head_is_static) {
  if (!mass || !head_is_static || n_heads < 0) return FK_ERR_ARG;
  if (alpha_permille < 0 || alpha_permille > 1000) return FK_ERR_CONFIG;
  for (int hd = 0; hd < n_heads; ++hd) {
    const double* m = mass + (int64_t)hd * 4;
    const double local = m[1] + m[2];          // generated chunk + transition frame
    const double window = m[0] - m[3];         // whole window minus the sink frames
    // a head whose mass lies entirely on the sink frames counts as static
    head_is_static[hd] = (window <= 0.0 || local * 1000.0 > (double)alpha_permille * window) ? 1 : 0;
  }
  return FK_OK;
}

fk_status fk_stream_read(const void* src, size_t bytes, void* stream) {
  if (!src || !aligned16(src) || (bytes & 15u)) return FK_ERR_ARG;
  if (bytes == 0) return FK_OK;
  if (!is_device_ptr(src)) return FK_ERR_ARG;
  return launch_stream_read(src, (int64_t)bytes, static_cast<cudaStream_t>(stream)) == cudaSuccess
             ? FK_OK
             : FK_ERR_CUDA;
}

fk_status fk_wait_selftest(fk_handle* h, int limit_us, void* stream) {
  if (!h) return FK_ERR_ARG;
  if (limit_us < 1 || limit_us > 2000000) return FK_ERR_ARG;
  FK_CUDA(cudaSetDevice(h->dev));
  return launch_wait_selftest((uint64_t)limit_us * 1000ull, h->status,
                              static_cast<cudaStream_t>(stream)) == cudaSuccess
             ? FK_OK
             : FK_ERR_CUDA;
}

fk_status fk_set_host_overlap(fk_handle* h, int on) {
  if (!h) return FK_ERR_ARG;
  h->host_overlap = on != 0;
  return FK_OK;
}

fk_status fk_wait_outputs(fk_handle* h, void* stream) {
  if (!h) return FK_ERR_ARG;
  FK_CUDA(cudaSetDevice(h->dev));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  for (int sl = 0; sl < 2; ++sl)
    if (h->o_pending[sl]) FK_CUDA(cudaStreamWaitEvent(s, h->o_copied[sl], 0));
  return FK_OK;
}

int fk_abi_version(void) { return 4; }

const char* fk_status_str(fk_status s) {
  switch (s) {
    case FK_OK: return "ok";
    case FK_ERR_CONFIG: return "invalid configuration";
    case FK_ERR_ARG: return "invalid argument";
    case FK_ERR_STATE: return "call out of order";
    case FK_ERR_FULL: return "history capacity exceeded";
    case FK_ERR_RANGE: return "scoring precondition violated (token squared key norm > 2^23)";
    case FK_ERR_TIMEOUT: return "bounded device wait expired";
    case FK_ERR_CUDA: return "CUDA error";
    case FK_ERR_NOMEM: return "out of device memory";
  }
  return "unknown status";
}

fk_status fk_validate_config(const fk_config* c) {
  if (!c || !c->head_is_static) return FK_ERR_ARG;
  if (c->n_layers < 1 || c->n_layers > kMaxLayers) return FK_ERR_CONFIG;
  if (c->n_heads < 1 || c->n_heads > kMaxHeads) return FK_ERR_CONFIG;
  if (c->head_dim != 64 && c->head_dim != 128) return FK_ERR_CONFIG;
  if (c->tokens_per_frame < 1 || c->n_segments < 1 || c->tokens_per_frame % c->n_segments)
    return FK_ERR_CONFIG;
  if (c->frames_per_chunk < 1 || c->n_sink_frames < 0 || c->window_frames < 0) return FK_ERR_CONFIG;
  if (c->keep_budget_permille < 0 || c->keep_budget_permille > 1000) return FK_ERR_CONFIG;
  if (c->select_scope != FK_SCOPE_PER_FRAME && c->select_scope != FK_SCOPE_POOLED) return FK_ERR_CONFIG;
  if (c->score_source != FK_SCORE_PER_HEAD && c->score_source != FK_SCORE_LAYER0_POOLED)
    return FK_ERR_CONFIG;
  if (c->incremental != 0 && c->incremental != 1) return FK_ERR_CONFIG;
  if (c->window_frames == 0 && c->max_history_frames < 1) return FK_ERR_CONFIG;
  if (c->selection < FK_SELECT_SIMILARITY || c->selection > FK_SELECT_RANDOM) return FK_ERR_CONFIG;
  if (c->selection == FK_SELECT_UNIFORM && c->select_scope != FK_SCOPE_PER_FRAME) return FK_ERR_CONFIG;
  if (c->static_drop_anchor != 0 && c->static_drop_anchor != 1) return FK_ERR_CONFIG;
  if (c->attn_precision != FK_ATTN_BF16 && c->attn_precision != FK_ATTN_FP8_QK &&
      c->attn_precision != FK_ATTN_FP8)
    return FK_ERR_CONFIG;
  if (c->attn_precision != FK_ATTN_BF16 && c->head_dim != 128) return FK_ERR_CONFIG;
  const int64_t cf = (int64_t)c->frames_per_chunk * c->tokens_per_frame;
  if (cf > (1 << 24) || (int64_t)c->tokens_per_frame * c->head_dim > (1 << 28)) return FK_ERR_CONFIG;
  // 16-byte granules of one chunk (all heads) are indexed with 32-bit integers
  if (cf * c->n_heads * (c->head_dim / 8) >= ((int64_t)1 << 31)) return FK_ERR_CONFIG;
  const int64_t cap = c->window_frames > 0 ? c->window_frames
                                           : std::max(0, c->max_history_frames - c->n_sink_frames);
  if (cap > 4096 || c->n_sink_frames > 4096) return FK_ERR_CONFIG;
  return FK_OK;
}

fk_status fk_create(const fk_config* cfg, fk_handle** out) {
  if (!out) return FK_ERR_ARG;
  *out = nullptr;
  fk_status st = fk_validate_config(cfg);
  if (st != FK_OK) return st;
  fk_handle* h = new (std::nothrow) fk_handle();
  if (!h) return FK_ERR_NOMEM;
  h->cfg = *cfg;
  h->L = cfg->n_layers;
  h->H = cfg->n_heads;
  h->D = cfg->head_dim;
  h->F = cfg->tokens_per_frame;
  h->C = cfg->frames_per_chunk;
  h->S = cfg->n_sink_frames;
  h->W = cfg->window_frames;
  h->n = cfg->n_segments;
  h->b = cfg->keep_budget_permille;
  h->scope = cfg->select_scope;
  h->source = cfg->score_source;
  h->incremental = cfg->incremental;
  h->max_hist = cfg->max_history_frames;
  h->dev = cfg->device;
  h->seg = h->F / h->n;
  h->CF = h->C * h->F;
  h->static_map.assign(cfg->head_is_static, cfg->head_is_static + (size_t)h->L * h->H);
  h->cfg.head_is_static = h->static_map.data();
  h->cap_nonsink = h->W > 0 ? h->W : std::max(0, h->max_hist - h->S);
  if (h->cap_nonsink < 1) h->cap_nonsink = 1;
  h->ring_slots = h->S + h->cap_nonsink;
  h->selection = cfg->selection;
  h->select_seed = cfg->select_seed;
  h->drop_anchor = cfg->static_drop_anchor != 0;
  h->precision = cfg->attn_precision;
  h->fp8 = cfg->attn_precision != FK_ATTN_BF16;
  h->fp8pv = cfg->attn_precision == FK_ATTN_FP8;
  h->k_frame = h->selection == FK_SELECT_ALL ? h->n : (h->b * h->n) / 1000;
  h->kmax = std::max(1, keep_total(h, h->cap_nonsink - 1));
  h->chunks = (h->seg + kScoreTokensPerCta - 1) / kScoreTokensPerCta;
  h->max_run = h->cap_nonsink;
  h->heads.resize((size_t)h->L * h->H);
  h->layers.resize(h->L);

  auto fail = [&](fk_status s) {
    fk_destroy(h);
    return s;
  };
  if (cudaSetDevice(h->dev) != cudaSuccess) {
    cudaGetLastError();
    return fail(FK_ERR_CUDA);
  }
  if (!get_encode()) return fail(FK_ERR_CUDA);
  if (attention_prepare(h->D) != cudaSuccess) return fail(FK_ERR_CUDA);
  if (score_prepare(h->D, h->cap_nonsink, h->n, &h->score_ctas) != cudaSuccess) return fail(FK_ERR_CUDA);

  // heads: roles, view rows, targets
  int n_dynamic = 0;
  for (int l = 0; l < h->L; ++l)
    for (int hd = 0; hd < h->H; ++hd) {
      HeadBuf& hb = h->heads[l * h->H + hd];
      hb.is_static = h->static_map[l * h->H + hd] != 0;
      hb.retains = !hb.is_static || (h->source == FK_SCORE_LAYER0_POOLED && l == 0);
      const int64_t rows = hb.is_static
                               ? (int64_t)h->CF + (int64_t)h->S * h->F + h->F
                               : (int64_t)h->CF + (int64_t)h->S * h->F + (int64_t)h->kmax * h->seg + h->F;
      hb.view_rows = (int)round_up(rows, kViewAlignRows);
      hb.row_base = h->view_rows_total;
      h->view_rows_total += hb.view_rows;
      n_dynamic += !hb.is_static;
    }
  if (h->view_rows_total >= (int64_t)1 << 31) return fail(FK_ERR_CONFIG);
  if (h->source == FK_SCORE_LAYER0_POOLED) {
    h->targets.push_back({0, 0, h->H});
    h->target_layer.push_back(0);
    for (int hd = 0; hd < h->H; ++hd) h->score_items.push_back({nullptr, 0, 0});
    for (auto& hb : h->heads)
      if (!hb.is_static) hb.target = 0;
  } else {
    for (int l = 0; l < h->L; ++l)
      for (int hd = 0; hd < h->H; ++hd) {
        HeadBuf& hb = h->heads[l * h->H + hd];
        if (hb.is_static) continue;
        hb.target = (int)h->targets.size();
        h->targets.push_back({l, (int)h->score_items.size(), 1});
        h->target_layer.push_back(l);
        h->score_items.push_back({nullptr, l, hb.target});
      }
  }
  h->layer_items.assign(h->L, {0, 0});   // score items are grouped by ascending layer
  for (size_t y = 0; y < h->score_items.size(); ++y) {
    auto& li = h->layer_items[h->score_items[y].layer];
    if (li.second == 0) li.first = (int)y;
    ++li.second;
  }

  // allocations
  void* p = nullptr;
  const size_t view_bytes = (size_t)h->view_rows_total * h->D * 2;
  if ((st = dev_alloc(h, view_bytes, &p)) != FK_OK) return fail(st);
  h->viewK = static_cast<bf16*>(p);
  if ((st = dev_alloc(h, view_bytes, &p)) != FK_OK) return fail(st);
  h->viewV = static_cast<bf16*>(p);
  if (h->fp8pv) {
    if ((st = dev_alloc(h, view_bytes / 2, &p)) != FK_OK) return fail(st);
    h->viewV8 = static_cast<uint8_t*>(p);
  }
  if (h->fp8) {
    if ((st = dev_alloc(h, view_bytes / 2, &p)) != FK_OK) return fail(st);
    h->viewK8 = static_cast<uint8_t*>(p);
  }
  size_t n_ret = 0;
  for (auto& hb : h->heads) n_ret += hb.retains;
  const size_t ring_elems = (size_t)h->ring_slots * h->F * h->D;
  bf16* pages = nullptr;
  if (n_ret) {
    if ((st = dev_alloc(h, n_ret * ring_elems * 2 * 2, &p)) != FK_OK) return fail(st);
    pages = static_cast<bf16*>(p);
  }
  size_t ri = 0;
  for (auto& hb : h->heads) {
    hb.viewK = h->viewK + hb.row_base * h->D;
    hb.viewV = h->viewV + hb.row_base * h->D;
    if (hb.retains) {
      hb.pageK = pages + (2 * ri) * ring_elems;
      hb.pageV = pages + (2 * ri + 1) * ring_elems;
      ++ri;
    }
  }
  const size_t nt = std::max<size_t>(1, h->targets.size());
  if ((st = dev_alloc(h, nt * h->ring_slots * h->n * sizeof(float), &p)) != FK_OK) return fail(st);
  h->scores = static_cast<float*>(p);
  if ((st = dev_alloc(h, nt * h->kmax * sizeof(int), &p)) != FK_OK) return fail(st);
  h->kept = static_cast<int*>(p);
  const size_t n_items = std::max<size_t>(1, h->score_items.size());
  h->sums_bytes = nt * h->max_run * h->n * 2 * sizeof(unsigned long long);
  if ((st = dev_alloc(h, h->sums_bytes, &p)) != FK_OK) return fail(st);
  h->sums = static_cast<unsigned long long*>(p);
  if ((st = dev_alloc(h, 256, &p)) != FK_OK) return fail(st);
  h->status = static_cast<int*>(p);
  const size_t chunk_bytes = (size_t)h->CF * h->H * h->D * 2;
  for (int sl = 0; sl < 2; ++sl) {
    for (int i = 0; i < 2; ++i) {
      if ((st = dev_alloc(h, chunk_bytes, &p)) != FK_OK) return fail(st);
      h->st_kv.buf[sl][i] = static_cast<bf16*>(p);
    }
    if ((st = dev_alloc(h, chunk_bytes, &p)) != FK_OK) return fail(st);
    h->st_q.buf[sl][0] = static_cast<bf16*>(p);
  }
  for (int sl = 0; sl < 2; ++sl) {
    if ((st = dev_alloc(h, chunk_bytes, &p)) != FK_OK) return fail(st);
    h->stage_o[sl] = static_cast<bf16*>(p);
    if (cudaEventCreateWithFlags(&h->o_ready[sl], cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&h->o_copied[sl], cudaEventDisableTiming) != cudaSuccess) {
      cudaGetLastError();
      return fail(FK_ERR_CUDA);
    }
  }
  if ((st = dev_alloc(h, (size_t)kMaxKvSplits * h->CF * h->H * h->D * sizeof(float), &p)) != FK_OK)
    return fail(st);
  h->part_o = static_cast<float*>(p);
  if ((st = dev_alloc(h, (size_t)kMaxKvSplits * h->CF * h->H * sizeof(float2), &p)) != FK_OK)
    return fail(st);
  h->part_ml = static_cast<float2*>(p);
  if (cudaDeviceGetAttribute(&h->n_sms, cudaDevAttrMultiProcessorCount, h->dev) != cudaSuccess) {
    cudaGetLastError();
    return fail(FK_ERR_CUDA);
  }
  h->split_keys.assign(h->L, {});
  h->split_choice.assign(h->L, 1);
  h->stage_frames = h->C;
  for (Staging* sg : {&h->st_kv, &h->st_q})
    for (int sl = 0; sl < 2; ++sl)
      if (cudaEventCreateWithFlags(&sg->ready[sl], cudaEventDisableTiming) != cudaSuccess ||
          cudaEventCreateWithFlags(&sg->freed[sl], cudaEventDisableTiming) != cudaSuccess) {
        cudaGetLastError();
        return fail(FK_ERR_CUDA);
      }
  if (cudaStreamCreateWithFlags(&h->copy_stream, cudaStreamNonBlocking) != cudaSuccess ||
      cudaStreamCreateWithFlags(&h->copy_out_stream, cudaStreamNonBlocking) != cudaSuccess) {
    cudaGetLastError();
    return fail(FK_ERR_CUDA);
  }

  // static device tables
  if (h->source == FK_SCORE_LAYER0_POOLED) {
    for (int hd = 0; hd < h->H; ++hd) h->score_items[hd].pagesK = h->heads[hd].pageK;
  } else {
    for (auto& si : h->score_items) {
      for (int hd = 0; hd < h->H; ++hd) {
        const HeadBuf& hb = h->heads[si.layer * h->H + hd];
        if (hb.target == si.target) si.pagesK = hb.pageK;
      }
    }
  }
  for (int l = 0; l < h->L; ++l)
    for (int hd = 0; hd < h->H; ++hd) {
      const HeadBuf& hb = h->heads[l * h->H + hd];
      if (hb.is_static) continue;
      h->compact_items.push_back({hb.pageK, hb.pageV, hb.viewK, hb.viewV, l, hb.target,
                                  h->fp8 ? h->viewK8 + hb.row_base * h->D : nullptr,
                                  h->fp8pv ? h->viewV8 + hb.row_base * h->D : nullptr});
    }
  auto upload = [&](const void* src, size_t bytes, void** dst) -> fk_status {
    fk_status s2 = dev_alloc(h, std::max<size_t>(bytes, 16), dst);
    if (s2 != FK_OK) return s2;
    if (bytes && cudaMemcpy(*dst, src, bytes, cudaMemcpyHostToDevice) != cudaSuccess) return FK_ERR_CUDA;
    return FK_OK;
  };
  if ((st = upload(h->score_items.data(), h->score_items.size() * sizeof(ScoreItem), &p)) != FK_OK)
    return fail(st);
  h->d_score_items = static_cast<ScoreItem*>(p);
  if ((st = upload(h->targets.data(), h->targets.size() * sizeof(SelectTarget), &p)) != FK_OK)
    return fail(st);
  h->d_targets = static_cast<SelectTarget*>(p);
  if ((st = upload(h->compact_items.data(), h->compact_items.size() * sizeof(CompactItem), &p)) != FK_OK)
    return fail(st);
  h->d_compact_items = static_cast<CompactItem*>(p);

  if ((st = encode_2d(&h->tmK, h->viewK, h->view_rows_total, h->D)) != FK_OK) return fail(st);
  if ((st = encode_2d(&h->tmV, h->viewV, h->view_rows_total, h->D)) != FK_OK) return fail(st);
  if (h->fp8 && (st = encode_2d(&h->tmK8, h->viewK8, h->view_rows_total, h->D, true)) != FK_OK)
    return fail(st);
  if (h->fp8pv && (st = encode_2d(&h->tmV8, h->viewV8, h->view_rows_total, h->D, true)) != FK_OK)
    return fail(st);
  if (cudaDeviceSynchronize() != cudaSuccess) return fail(FK_ERR_CUDA);
  for (int l = 0; l < h->L; ++l) update_lengths(h, l);
  *out = h;
  return FK_OK;
}

void fk_destroy(fk_handle* h) {
  if (!h) return;
  cudaSetDevice(h->dev);
  cudaDeviceSynchronize();
  for (auto& r : h->prof_pending) {
    cudaEventDestroy(r.a);
    cudaEventDestroy(r.b);
  }
  for (auto e : h->ev_free) cudaEventDestroy(e);
  for (Staging* sg : {&h->st_kv, &h->st_q})
    for (int sl = 0; sl < 2; ++sl) {
      if (sg->ready[sl]) cudaEventDestroy(sg->ready[sl]);
      if (sg->freed[sl]) cudaEventDestroy(sg->freed[sl]);
    }
  if (h->copy_stream) cudaStreamDestroy(h->copy_stream);
  if (h->copy_out_stream) cudaStreamDestroy(h->copy_out_stream);
  for (int sl = 0; sl < 2; ++sl) {
    if (h->o_ready[sl]) cudaEventDestroy(h->o_ready[sl]);
    if (h->o_copied[sl]) cudaEventDestroy(h->o_copied[sl]);
  }
  for (void* p : h->allocs) cudaFree(p);
  cudaGetLastError();
  delete h;
}

static fk_status check_layer(const fk_handle* h, int layer) {
  if (!h) return FK_ERR_ARG;
  if (layer < 0 || layer >= h->L) return FK_ERR_ARG;
  return FK_OK;
}

fk_status fk_append_frames(fk_handle* h, int layer, const void* K, const void* V, int n_frames,
                           void* stream) {
  fk_status st = check_layer(h, layer);
  if (st != FK_OK) return st;
  if (n_frames < 0 || (n_frames > 0 && (!K || !V))) return FK_ERR_ARG;
  if (n_frames > 0 && (!aligned16(K) || !aligned16(V))) return FK_ERR_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  FK_CUDA(cudaSetDevice(h->dev));
  LayerState& ls = h->layers[layer];
  const int extra = ls.has_current ? h->C : 0;
  if (h->W == 0 && ls.nh + extra + n_frames > h->max_hist) return FK_ERR_FULL;
  if ((st = update_current(h, layer, true, nullptr, nullptr, s)) != FK_OK) return st;
  const bool dev_in = n_frames > 0 && is_device_ptr(K) && is_device_ptr(V);
  const size_t frame_bytes = (size_t)h->F * h->H * h->D * 2;
  for (int f0 = 0; f0 < n_frames;) {
    const int nf = dev_in ? n_frames : (int)std::min<int64_t>(h->stage_frames, n_frames - f0);
    const bf16* k = static_cast<const bf16*>(K) + (size_t)f0 * frame_bytes / 2;
    const bf16* v = static_cast<const bf16*>(V) + (size_t)f0 * frame_bytes / 2;
    if (!dev_in) {   // staging slot 0, in order on `s` (see the freed events below)
      FK_CUDA(cudaMemcpyAsync(h->st_kv.buf[0][0], k, nf * frame_bytes, cudaMemcpyHostToDevice, s));
      FK_CUDA(cudaMemcpyAsync(h->st_kv.buf[0][1], v, nf * frame_bytes, cudaMemcpyHostToDevice, s));
      k = h->st_kv.buf[0][0];
      v = h->st_kv.buf[0][1];
    }
    if ((st = push_history(h, layer, k, v, nf, s)) != FK_OK) return st;
    f0 += nf;
  }
  if (n_frames > 0 && !dev_in)   // later overlapped copies into either slot wait for this use
    for (int sl = 0; sl < 2; ++sl) FK_CUDA(cudaEventRecord(h->st_kv.freed[sl], s));
  ls.dirty = true;
  return FK_OK;
}

fk_status fk_append_chunk(fk_handle* h, int layer, const void* K, const void* V, void* stream) {
  fk_status st = check_layer(h, layer);
  if (st != FK_OK) return st;
  if (!K || !V || !aligned16(K) || !aligned16(V)) return FK_ERR_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  FK_CUDA(cudaSetDevice(h->dev));
  if ((st = update_current(h, layer, true, K, V, s)) != FK_OK) return st;
  h->layers[layer].dirty = true;
  return FK_OK;
}

fk_status fk_set_current(fk_handle* h, int layer, const void* K, const void* V, void* stream) {
  fk_status st = check_layer(h, layer);
  if (st != FK_OK) return st;
  if (!K || !V || !aligned16(K) || !aligned16(V)) return FK_ERR_ARG;
  FK_CUDA(cudaSetDevice(h->dev));
  return update_current(h, layer, false, K, V, static_cast<cudaStream_t>(stream));
}

fk_status fk_compress(fk_handle* h, void* stream) {
  if (!h) return FK_ERR_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  FK_CUDA(cudaSetDevice(h->dev));
  bool any = false;
  for (auto& ls : h->layers) any |= ls.dirty;
  if (!any) return FK_OK;
  const bool pooled_src = h->source == FK_SCORE_LAYER0_POOLED;
  if (pooled_src) {
    for (int l = 1; l < h->L; ++l)
      if (h->layers[l].nh != h->layers[0].nh) return FK_ERR_STATE;
  }
  ScoreArgs sa{};
  CompactArgs ca{};
  bool any_run = false, any_compact = false, clear_sums = false;
  // incremental compaction needs kept sets that never change once decided: per-frame scope
  const bool inc_compact = h->incremental && h->scope == FK_SCOPE_PER_FRAME;
  std::vector<int> keep_of(h->L, 0);
  for (int l = 0; l < h->L; ++l) {
    LayerState& ls = h->layers[l];
    const Roles r = roles_of(h, ls.nh);
    const int keep = keep_total(h, r.n_scoreable);
    // scoring run of the layer whose keys score (every layer per head; layer 0 pooled)
    const bool scores_here = pooled_src ? l == 0 : true;
    if (ls.dirty && scores_here && h->selection != FK_SELECT_SIMILARITY) {
      // comparison rules: no scoring; the selection kernel ranks the whole window by the
      // rule's values
      if (r.n_scoreable > 0) {
        sa.run[l] = {r.t_lo, r.n_scoreable + 1, 0, r.n_scoreable + 1};
        any_run = true;
      }
    } else if (ls.dirty && scores_here) {
      const int t_first = h->incremental ? std::max(r.t_lo, ls.scored_upto) : r.t_lo;
      const int last_t = r.t_lo + r.n_scoreable - 1;
      if (r.n_scoreable > 0 && t_first <= last_t) {
        // the chunk the last append retired, [nh - C, nh), may still be in flight
        const int n_run = last_t + 2 - t_first;
        int n_read = n_run;
        if (ls.fuse_state == 1 && ls.fuse_t_first == t_first && ls.fuse_end == t_first + n_run)
          n_read = ls.fuse_n_read;   // the current-chunk kernel formed the rest of the sums
        else if (ls.fuse_state != 0)
          clear_sums = true;         // partial sums that match no run: clear, rescore all
        sa.run[l] = {t_first, n_run, std::max(0, ls.nh - h->C), n_read};
        any_run = true;
      } else if (ls.fuse_state != 0) {
        clear_sums = true;
      }
      ls.scored_upto = r.anchor >= 0 ? r.anchor : ls.scored_upto;
    }
    if (scores_here) ls.fuse_state = 0;
    sa.t_lo[l] = r.t_lo;
    sa.n_scoreable[l] = r.n_scoreable;
    sa.n_keep[l] = keep;
    keep_of[l] = keep;
    ca.active[l] = ls.dirty ? 1 : 0;
    if (!ls.dirty) continue;
    if (inc_compact) {
      // frames below the window leave the ring; the newly decided frames are appended.  A
      // frame leaves only once the window is full, and then the ring is full again after the
      // append, so the valid slots are always [0, count) or all kmax: one contiguous key range
      const int t_hi = r.t_lo + r.n_scoreable;
      if (r.t_lo > ls.ring_first) {
        const int gone = std::min(r.t_lo, ls.ring_end) - ls.ring_first;
        if (gone > 0)
          ls.ring_head = (int)(((int64_t)ls.ring_head + (int64_t)gone * h->k_frame) % h->kmax);
        ls.ring_first = r.t_lo;
        ls.ring_end = std::max(ls.ring_end, r.t_lo);
      }
      const int n_add = std::max(0, t_hi - ls.ring_end);
      ca.n_kept_copy[l] = n_add * h->k_frame;
      ca.kp0[l] = (ls.ring_end - r.t_lo) * h->k_frame;
      ca.rp0[l] = (int)(((int64_t)ls.ring_head + (int64_t)(ls.ring_end - ls.ring_first) * h->k_frame) % h->kmax);
      ls.ring_end = std::max(ls.ring_end, t_hi);
      if (ls.ring_head != 0 && keep != h->kmax) return FK_ERR_STATE;   // cannot happen (see above)
    } else {
      ca.n_kept_copy[l] = keep;
      ca.kp0[l] = 0;
      ca.rp0[l] = 0;
    }
    ca.max_units = std::max(ca.max_units, ca.n_kept_copy[l]);
  }
  for (const auto& ci : h->compact_items) any_compact |= ca.active[ci.layer] != 0;
  fk_status st;
  if (any_run) {
    sa.items = h->d_score_items;
    sa.targets = h->d_targets;
    sa.n_items = (int)h->score_items.size();
    sa.F = h->F;
    sa.D = h->D;
    sa.n_seg = h->n;
    sa.seg_len = h->seg;
    sa.chunks = h->chunks;
    sa.S = h->S;
    sa.cap_nonsink = h->cap_nonsink;
    sa.ring_slots = h->ring_slots;
    sa.max_run = h->max_run;
    sa.scope = h->scope;
    sa.k_frame = h->k_frame;
    sa.kmax = h->kmax;
    sa.sums = h->sums;
    sa.max_ctas = h->score_ctas;
    // active layers in ascending order with the start of their frame-chunks in the
    // flattened (layer, item, segment, chunk, frame) range; items are grouped by layer
    long long units = 0;
    for (int l = 0; l < h->L; ++l) {
      if (clear_sums) sa.run[l].n_read = sa.run[l].n_run;
      if (sa.run[l].n_read == 0 || h->layer_items[l].second == 0) continue;
      sa.act_layer[sa.n_active] = l;
      sa.act_first_item[sa.n_active] = h->layer_items[l].first;
      sa.act_start[sa.n_active] = units;
      units += (long long)h->layer_items[l].second * h->n * h->chunks * sa.run[l].n_read;
      ++sa.n_active;
    }
    sa.total_units = units;
    sa.scores = h->scores;
    sa.kept = h->kept;
    sa.status = h->status;
    sa.rule = h->selection;
    sa.seed = h->select_seed;
    if (clear_sums)
      FK_CUDA(cudaMemsetAsync(h->sums, 0, h->sums_bytes, s));
    if (h->selection == FK_SELECT_SIMILARITY && units > 0 &&
        (st = launch(h, s, FK_KERNEL_SCORE, [&] { launch_score(sa, s); })) != FK_OK)
      return st;
    const int nt = (int)h->targets.size();
    if ((st = launch(h, s, FK_KERNEL_SELECT, [&] { launch_select(sa, nt, s); })) != FK_OK) return st;
  }
  if (any_compact && ca.max_units > 0) {
    ca.items = h->d_compact_items;
    ca.n_items = (int)h->compact_items.size();
    ca.F = h->F;
    ca.D = h->D;
    ca.n_seg = h->n;
    ca.seg_len = h->seg;
    ca.CF = h->CF;
    ca.S = h->S;
    ca.cap_nonsink = h->cap_nonsink;
    ca.kmax = h->kmax;
    const int64_t unit_bytes = (int64_t)h->seg * h->D * 2;
    ca.splits = (int)((unit_bytes + kCompactPiece - 1) / kCompactPiece);
    ca.units_per_cta = unit_bytes < kCompactPiece ? (int)(kCompactPiece / unit_bytes) : 1;
    ca.kept = h->kept;
    if ((st = launch(h, s, FK_KERNEL_COMPACT, [&] { launch_compact(ca, s); })) != FK_OK) return st;
  }
  for (int l = 0; l < h->L; ++l) {
    LayerState& ls = h->layers[l];
    if (!ls.dirty) continue;
    ls.n_keep = keep_of[l];
    ls.dirty = false;
    update_lengths(h, l);
  }
  return FK_OK;
}

fk_status fk_attend(fk_handle* h, int layer, const void* Q, void* O, void* stream) {
  fk_status st = check_layer(h, layer);
  if (st != FK_OK) return st;
  if (!Q || !O || !aligned16(Q) || !aligned16(O)) return FK_ERR_ARG;
  const LayerState& ls = h->layers[layer];
  if (!ls.has_current || ls.dirty) return FK_ERR_STATE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  FK_CUDA(cudaSetDevice(h->dev));
  const size_t bytes = (size_t)h->CF * h->H * h->D * 2;
  const bf16* q = nullptr;
  int slot = -1;
  if ((st = stage_inputs(h, h->st_q, Q, nullptr, bytes, s, &q, nullptr, &slot)) != FK_OK) return st;
  // a host output is staged and copied back on `stream` (measured faster than storing it
  // from the attention epilogue directly into pinned host memory)
  const bool copy_back = !is_device_ptr(O);
  const int osl = h->o_slot;
  bf16* o = static_cast<bf16*>(O);
  if (copy_back) {
    h->o_slot ^= 1;
    o = h->stage_o[osl];
    // the slot's previous copy-back (two host-output calls ago) must have read it
    if (h->o_pending[osl]) FK_CUDA(cudaStreamWaitEvent(s, h->o_copied[osl], 0));
  }
  int qm = q == h->q_cached[0] ? 0 : q == h->q_cached[1] ? 1 : -1;
  if (qm < 0) {
    qm = h->q_next;
    h->q_next ^= 1;
    if ((st = encode_q(&h->tmQ[qm], q, h->CF, h->H, h->D)) != FK_OK) return st;
    h->q_cached[qm] = q;
  }
  AttnArgs a{};
  a.O = o;
  a.Nq = h->CF;
  a.H = h->H;
  a.n_qtiles = (h->CF + 2 * kAttnBM - 1) / (2 * kAttnBM);   // CTA = two 128-row query tiles
  a.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)h->D));
  a.status = h->status;
  std::vector<int> order(h->H);
  for (int hd = 0; hd < h->H; ++hd) {
    const HeadBuf& hb = h->heads[layer * h->H + hd];
    a.row_base[hd] = (int)hb.row_base;
    a.n_keys[hd] = hb.is_static ? ls.len_static : ls.len_dynamic;
    order[hd] = hd;
  }
  std::stable_sort(order.begin(), order.end(),
                   [&](int x, int y) { return a.n_keys[x] > a.n_keys[y]; });
  for (int i = 0; i < h->H; ++i) a.head_of[i] = order[i];
  std::vector<int> keys(a.n_keys, a.n_keys + h->H);
  if (keys != h->split_keys[layer]) {
    h->split_choice[layer] = choose_kv_splits(h->n_sms, a.n_qtiles, h->CF, h->H, h->D, a.n_keys);
    h->split_keys[layer] = keys;
  }
  a.kv_splits = h->split_choice[layer];
  a.part_o = h->part_o;
  a.part_ml = h->part_ml;
  const int D = h->D;
  // FP8: the E4M3 keys (and, for P V, values) come from the view arenas' E4M3 copies; the kernel
  // quantizes Q
  const CUtensorMap& tk = h->fp8 ? h->tmK8 : h->tmK;
  const CUtensorMap& tv = h->fp8pv ? h->tmV8 : h->tmV;
  if ((st = launch(h, s, FK_KERNEL_ATTEND, [&] {
         launch_attention(D, h->precision, h->tmQ[qm], tk, tv, a, s);
         if (a.kv_splits > 1) launch_merge(D, a, s);
       })) != FK_OK)
    return st;
  if (a.kv_splits > 1) h->launches++;   // the merge pass
  if (slot >= 0) FK_CUDA(cudaEventRecord(h->st_q.freed[slot], s));
  if (copy_back) {
    if (h->host_overlap) {   // copy back off the caller's stream; fk_wait_outputs joins it
      FK_CUDA(cudaEventRecord(h->o_ready[osl], s));
      FK_CUDA(cudaStreamWaitEvent(h->copy_out_stream, h->o_ready[osl], 0));
      FK_CUDA(cudaMemcpyAsync(O, o, bytes, cudaMemcpyDeviceToHost, h->copy_out_stream));
      FK_CUDA(cudaEventRecord(h->o_copied[osl], h->copy_out_stream));
      h->o_pending[osl] = true;
    } else {
      FK_CUDA(cudaMemcpyAsync(O, o, bytes, cudaMemcpyDeviceToHost, s));
      h->o_pending[osl] = false;
    }
  }
  return FK_OK;
}

size_t fk_cache_bytes(const fk_handle* h) {
  if (!h) return 0;
  size_t bytes = 0;
  const size_t frame_bytes = (size_t)h->F * h->D * 2 * 2;   // K and V
  for (int l = 0; l < h->L; ++l) {
    const LayerState& ls = h->layers[l];
    const Roles r = roles_of(h, ls.nh);
    const int live_frames = r.n_sink + (ls.nh - r.lo > 0 ? ls.nh - r.lo : 0);
    for (int hd = 0; hd < h->H; ++hd) {
      const HeadBuf& hb = h->heads[l * h->H + hd];
      if (hb.retains) bytes += (size_t)live_frames * frame_bytes;
      const int rows = hb.is_static ? ls.len_static : ls.len_dynamic;
      bytes += (size_t)rows * h->D * (4 + (h->fp8 ? 1 : 0) + (h->fp8pv ? 1 : 0));   // bf16 K, V (+ E4M3)
    }
  }
  bytes += h->targets.size() * ((size_t)h->ring_slots * h->n * sizeof(float) + h->kmax * sizeof(int));
  return bytes;
}

size_t fk_reserved_bytes(const fk_handle* h) { return h ? h->reserved : 0; }

fk_status fk_key_count(const fk_handle* h, int layer, int head, int* n_keys) {
  fk_status st = check_layer(h, layer);
  if (st != FK_OK) return st;
  if (head < 0 || head >= h->H || !n_keys) return FK_ERR_ARG;
  const LayerState& ls = h->layers[layer];
  *n_keys = h->heads[layer * h->H + head].is_static ? ls.len_static : ls.len_dynamic;
  return FK_OK;
}

fk_status fk_get_kept(fk_handle* h, int layer, int head, int32_t* out, int capacity, int* n_out,
                      void* stream) {
  fk_status st = check_layer(h, layer);
  if (st != FK_OK) return st;
  if (head < 0 || head >= h->H || !n_out) return FK_ERR_ARG;
  const HeadBuf& hb = h->heads[layer * h->H + head];
  if (hb.is_static) {
    *n_out = 0;
    return FK_OK;
  }
  const int n = h->layers[layer].n_keep;
  *n_out = n;
  if (capacity < n || (n > 0 && !out)) return FK_ERR_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  FK_CUDA(cudaSetDevice(h->dev));
  if (n > 0)
    FK_CUDA(cudaMemcpyAsync(out, h->kept + (size_t)hb.target * h->kmax, n * sizeof(int),
                            cudaMemcpyDeviceToHost, s));
  FK_CUDA(cudaStreamSynchronize(s));
  return FK_OK;
}

fk_status fk_get_scores(fk_handle* h, int layer, int head, float* out, int capacity,
                        int* first_frame, int* n_frames, void* stream) {
  fk_status st = check_layer(h, layer);
  if (st != FK_OK) return st;
  if (head < 0 || head >= h->H || !first_frame || !n_frames) return FK_ERR_ARG;
  const HeadBuf& hb = h->heads[layer * h->H + head];
  const int sl = h->source == FK_SCORE_LAYER0_POOLED ? 0 : layer;
  const Roles r = roles_of(h, h->layers[sl].nh);
  *first_frame = r.t_lo;
  *n_frames = hb.is_static ? 0 : r.n_scoreable;
  if (hb.is_static || r.n_scoreable == 0) return FK_OK;
  if (!out || capacity < r.n_scoreable * h->n) return FK_ERR_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  FK_CUDA(cudaSetDevice(h->dev));
  std::vector<float> all((size_t)h->ring_slots * h->n);
  FK_CUDA(cudaMemcpyAsync(all.data(), h->scores + (size_t)hb.target * h->ring_slots * h->n,
                          all.size() * sizeof(float), cudaMemcpyDeviceToHost, s));
  FK_CUDA(cudaStreamSynchronize(s));
  for (int i = 0; i < r.n_scoreable; ++i) {
    const int slot = ring_slot(h, r.t_lo + i);
    std::memcpy(out + (size_t)i * h->n, all.data() + (size_t)slot * h->n, h->n * sizeof(float));
  }
  return FK_OK;
}

fk_status fk_sync_status(fk_handle* h, void* stream) {
  if (!h) return FK_ERR_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  FK_CUDA(cudaSetDevice(h->dev));
  fk_status st = fk_wait_outputs(h, stream);   // overlapped output copies complete too
  if (st != FK_OK) return st;
  int word = 0;
  FK_CUDA(cudaMemcpyAsync(&word, h->status, sizeof(int), cudaMemcpyDeviceToHost, s));
  FK_CUDA(cudaStreamSynchronize(s));
  if (word) FK_CUDA(cudaMemset(h->status, 0, sizeof(int)));
  if (word & kStatusTimeout) return FK_ERR_TIMEOUT;
  if (word & kStatusRange) return FK_ERR_RANGE;
  return FK_OK;
}

fk_status fk_profile_enable(fk_handle* h, int on) {
  if (!h) return FK_ERR_ARG;
  FK_CUDA(cudaSetDevice(h->dev));
  if (on && h->ev_free.empty() && h->prof_pending.empty()) {
    for (int i = 0; i < 1024; ++i) {
      cudaEvent_t e;
      FK_CUDA(cudaEventCreate(&e));
      h->ev_free.push_back(e);
    }
  }
  h->prof = on != 0;
  return FK_OK;
}

fk_status fk_profile_read(fk_handle* h, int kind, double* total_ms, int64_t* launches) {
  if (!h || kind < 0 || kind >= FK_KERNEL_KINDS || !total_ms || !launches) return FK_ERR_ARG;
  FK_CUDA(cudaSetDevice(h->dev));
  fk_status st = prof_collect(h);
  if (st != FK_OK) return st;
  *total_ms = h->prof_ms[kind];
  *launches = h->prof_n[kind];
  return FK_OK;
}

fk_status fk_profile_reset(fk_handle* h) {
  if (!h) return FK_ERR_ARG;
  fk_status st = prof_collect(h);
  if (st != FK_OK) return st;
  for (int k = 0; k < FK_KERNEL_KINDS; ++k) {
    h->prof_ms[k] = 0;
    h->prof_n[k] = 0;
  }
  return FK_OK;
}

int64_t fk_launch_count(const fk_handle* h) { return h ? h->launches : 0; }

}  // extern "C"
