// Segment-wise similarity scoring (Sec. 4.3, Eq. 3) and BottomK selection: the scoring kernel,
// then the selection kernel chained to it by programmatic dependent launch.
//
// Work unit: one frame-chunk, i.e. 32 tokens of one segment of one scored (layer, head) in
// one frame of the run.  The units of all scored heads, ordered (layer, item, segment,
// token chunk, frame), are split into equal contiguous ranges, one per CTA of a persistent
// grid, so every CTA streams the same number of key bytes (no partial last wave).  A range
// walks consecutive frames of a token chunk; thread 0 streams each frame-chunk (8 KB
// contiguous) with one bulk copy into a shared-memory ring completed on mbarriers, loading one
// extra frame at the range's start as the partner of its first pair; every other key byte is
// read once.  Per token it forms the score-contract quantities (fp32 channel dot in a fixed
// fma/butterfly order, scaled by 2^24 and truncated to int64, carried as two exact int32
// halves): the squared norm n_p(t) and the dot d_p(t-1, t).  Warp sums go into shared-memory
// int32 accumulators (at most 32 tokens per run, so no overflow) and each run adds them as
// int64 into the target's global int64 sums (exact integer adds, so the order is free); no
// CTA waits for another.  The selection kernel (one CTA per target) then finishes
// s = D / sqrt(N_t N_{t+1}) in IEEE double, stores the fp32 scores per frame slot, clears the
// sums, ranks the scoreable candidates by (score, segment id) and stream-compacts the kept
// segment ids with warp ballots and prefix sums.
#include <algorithm>
#include <mutex>

#include "fk_internal.h"

namespace fk {
namespace {

__device__ __forceinline__ uint32_t su32_shared(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ uint4 lds128(uint32_t smem) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "r"(smem) : "memory");
  return v;
}

__device__ __forceinline__ int ring_slot(int f, int S, int cap) {
  return f < S ? f : S + (f - S) % cap;
}

__device__ __forceinline__ float finish_score(long long dsum, long long n1, long long n2) {
  if (n1 == 0 || n2 == 0) return 0.0f;
  const double den = __dsqrt_rn(__dmul_rn(__ll2double_rn(n1), __ll2double_rn(n2)));
  return __double2float_rn(__ddiv_rn(__ll2double_rn(dsum), den));
}

constexpr uint64_t kWaitLimitNs = 2000000000ull;   // 2 s per wait

__device__ __forceinline__ uint64_t now_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" :: "r"(bar), "r"(count));
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" :: "r"(bar), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ bool mbar_test(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok) : "r"(bar), "r"(parity) : "memory");
  return ok != 0;
}
// bounded wait for the phase of parity `parity`; false when the limit expired
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity,
                                          uint64_t limit_ns = kWaitLimitNs) {
  if (mbar_test(bar, parity)) return true;
  const uint64_t t0 = now_ns();
  while (!mbar_test(bar, parity))
    if (now_ns() - t0 > limit_ns) return false;
  return true;
}
// one contiguous global -> shared copy on the TMA engine, completing on `bar`
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
               :: "r"(dst), "l"(src), "r"(bytes), "r"(bar) : "memory");
}
// programmatic dependent launch: let the next kernel of the stream start its prologue /
// wait until the previous kernel of the stream has completed and its writes are visible
// (both are no-ops for a launch without the programmatic attribute)
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// SplitMix64 (Steele, Lea and Flood, 2014): the 64-bit finaliser of a Weyl sequence.
__device__ __forceinline__ unsigned long long splitmix64(unsigned long long z) {
  z += 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// Ranking value of candidate (t, j) under a comparison rule (BottomK keeps the smallest):
// ALL 0 for every segment (with k = n all are kept); UNIFORM 0 on the k segments
// j = floor(i n / k), i < k, else 1; RANDOM a uniform value in [0, 1) with 24 random bits,
// SplitMix64 of seed * 2^40 + t * 2^20 + j.
__device__ __forceinline__ float rule_value(int rule, unsigned int seed, int t, int j, int n, int k) {
  if (rule == FK_SELECT_UNIFORM) {
    if (k <= 0) return 1.0f;
    const long long i = ((long long)j * k + n - 1) / n;     // smallest i with i n / k >= j
    return (i < k && (i * n) / k == j) ? 0.0f : 1.0f;
  }
  if (rule == FK_SELECT_RANDOM) {
    const unsigned long long key = ((unsigned long long)seed << 40) ^ ((unsigned long long)t << 20) ^
                                   (unsigned long long)j;
    return (float)(splitmix64(key) >> 40) * (1.0f / 16777216.0f);
  }
  return 0.0f;
}

// Up to this many segments per frame the per-frame ranking compares every pair; above it
// (token-level rules) each frame is sorted in shared memory.
constexpr int kRankDirect = 64;
__host__ __device__ constexpr int select_sort_len(int n) {   // next power of two >= n
  int p = 1;
  while (p < n) p <<= 1;
  return p;
}
__host__ __device__ constexpr size_t select_sort_off(int max_run, int n) {   // 8-byte aligned
  return ((size_t)max_run * n * sizeof(float) + 7) / 8 * 8;
}

// BottomK of one frame with many segments (token-level rules): sort (value, id) keys in
// shared memory (bitonic), flag the k smallest ids, write them in ascending id order as
// frame-t segment ids into out[0 .. min(k, bound)).  Block-uniform arguments.
__device__ void sort_select_frame(const float* vals, int n, int k, int t, int* out, int bound,
                                  unsigned long long* key, int* flag, int* warp_tot, int* base_off) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int P = select_sort_len(n);
  for (int i = threadIdx.x; i < P; i += blockDim.x) {
    unsigned long long kv = ~0ull;
    if (i < n) {
      float v = vals[i];
      if (v == 0.0f) v = 0.0f;                       // -0 ranks as +0
      const uint32_t u = __float_as_uint(v);
      const uint32_t ord = (u & 0x80000000u) ? ~u : (u | 0x80000000u);   // order-preserving
      kv = ((unsigned long long)ord << 32) | (unsigned)i;
    }
    key[i] = kv;
  }
  for (int j = threadIdx.x; j < n; j += blockDim.x) flag[j] = 0;
  __syncthreads();
  for (int size = 2; size <= P; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = threadIdx.x; i < P / 2; i += blockDim.x) {
        const int lo = 2 * stride * (i / stride) + (i % stride), hi = lo + stride;
        const unsigned long long x = key[lo], y = key[hi];
        if ((x > y) == ((lo & size) == 0)) {
          key[lo] = y;
          key[hi] = x;
        }
      }
      __syncthreads();
    }
  }
  for (int i = threadIdx.x; i < k && i < n; i += blockDim.x) flag[(int)(key[i] & 0xFFFFFFFFu)] = 1;
  if (threadIdx.x == 0) *base_off = 0;
  __syncthreads();
  for (int b0 = 0; b0 < n; b0 += blockDim.x) {
    const int j = b0 + threadIdx.x;
    const bool keep = j < n && flag[j];
    const unsigned mask = __ballot_sync(0xffffffffu, keep);
    if (lane == 0) warp_tot[warp] = __popc(mask);
    __syncthreads();
    int woff = *base_off;
    for (int w = 0; w < warp; ++w) woff += warp_tot[w];
    const int pos = woff + __popc(mask & ((1u << lane) - 1u));
    if (keep && pos < bound) out[pos] = t * n + j;
    __syncthreads();
    if (threadIdx.x == 0) {
      int tot = 0;
      for (int w = 0; w < (int)(blockDim.x >> 5); ++w) tot += warp_tot[w];
      *base_off += tot;
    }
    __syncthreads();
  }
}

// Selection kernel for a comparison rule with many segments per frame (per-frame scope): one
// CTA per (target, frame of the window); the rule's values need no scores, so the frames are
// independent.
__global__ void __launch_bounds__(kSelectThreads) select_frames_kernel(const ScoreArgs a) {
  extern __shared__ float vals[];
  __shared__ int warp_tot[kSelectThreads / 32];
  __shared__ int base_off;
  const int tgi = blockIdx.x, f = blockIdx.y;
  const int l = a.targets[tgi].layer;
  pdl_trigger();
  pdl_wait();
  if (a.run[l].n_run < 2 || f >= a.n_scoreable[l]) return;
  const int n = a.n_seg, k = a.k_frame, t = a.t_lo[l] + f;
  float* sc = a.scores + (int64_t)tgi * a.ring_slots * n + (int64_t)ring_slot(t, a.S, a.cap_nonsink) * n;
  for (int j = threadIdx.x; j < n; j += blockDim.x) {
    const float v = rule_value(a.rule, a.seed, t, j, n, k);
    vals[j] = v;
    sc[j] = v;
  }
  unsigned long long* key = reinterpret_cast<unsigned long long*>(
      reinterpret_cast<uint8_t*>(vals) + ((size_t)n * sizeof(float) + 7) / 8 * 8);
  int* flag = reinterpret_cast<int*>(key + select_sort_len(n));
  __syncthreads();
  sort_select_frame(vals, n, k, t, a.kept + (int64_t)tgi * a.kmax + (int64_t)f * k,
                    a.n_keep[l] - f * k, key, flag, warp_tot, &base_off);
}

// Selection kernel: one CTA per selection target.  Finishes the pairs (t, t+1) scored by
// this launch from the target's int64 sums, clears the sums for the next launch, then
// BottomK over the scoreable frames compacted in ascending segment-id order; the window's
// scores are staged in shared memory in candidate order (t - t_lo)*n + j.
__global__ void __launch_bounds__(kSelectThreads) select_kernel(const ScoreArgs a) {
  extern __shared__ float ssc[];
  __shared__ int warp_tot[kSelectThreads / 32];
  __shared__ int base_off;
  const int tgi = blockIdx.x;
  const SelectTarget tg = a.targets[tgi];
  const int l = tg.layer;
  const LayerRun run = a.run[l];
  pdl_trigger();
  // every CTA waits, even one with nothing to do: this kernel's completion then implies the
  // completion of the kernels before it, which the next programmatic launch relies on
  pdl_wait();
  if (run.n_run < 2) return;
  const int n = a.n_seg;
  const int nT = a.n_scoreable[l];
  const int M = nT * n;
  const int t_lo = a.t_lo[l];
  float* sc = a.scores + (int64_t)tgi * a.ring_slots * n;
  unsigned long long* sums = a.sums + (int64_t)tgi * a.max_run * n * 2;
  if (a.rule != FK_SELECT_SIMILARITY) {
    // comparison rules: the ranking values come from the rule, not from scores
    for (int idx = threadIdx.x; idx < M; idx += blockDim.x) {
      const int t = t_lo + idx / n, jj = idx - (idx / n) * n;
      const float v = rule_value(a.rule, a.seed, t, jj, n, a.k_frame);
      ssc[idx] = v;
      sc[ring_slot(t, a.S, a.cap_nonsink) * n + jj] = v;
    }
    __syncthreads();
  } else {
  // 1. finish: s = D / sqrt(N_t N_{t+1}) in IEEE double, stored per frame slot and staged
  //    for the ranking when the frame is in the window
  const int pairs = (run.n_run - 1) * n;
  for (int idx = threadIdx.x; idx < pairs; idx += blockDim.x) {
    const int k = idx / n, j = idx - k * n;
    const unsigned long long N1 = sums[((int64_t)k * n + j) * 2];
    const unsigned long long N2 = sums[((int64_t)(k + 1) * n + j) * 2];
    const unsigned long long Dd = sums[((int64_t)(k + 1) * n + j) * 2 + 1];
    const int t = run.t_first + k;
    const float v = finish_score((long long)Dd, (long long)N1, (long long)N2);
    sc[ring_slot(t, a.S, a.cap_nonsink) * n + j] = v;
    if (t >= t_lo && t < t_lo + nT) ssc[(t - t_lo) * n + j] = v;
  }
  // window frames scored by an earlier launch (incremental scoring)
  for (int idx = threadIdx.x; idx < M; idx += blockDim.x) {
    const int t = t_lo + idx / n, jj = idx - (idx / n) * n;
    if (t < run.t_first) ssc[idx] = sc[ring_slot(t, a.S, a.cap_nonsink) * n + jj];
  }
  __syncthreads();   // every sum has been read
  for (int i = threadIdx.x; i < run.n_run * n * 2; i += blockDim.x) sums[i] = 0ull;
  }

  // 2. BottomK: rank by (score, segment id) within the frame (per-frame scope) or over the
  //    whole window (pooled scope), then stream-compact with warp ballots
  const int K = a.n_keep[l];
  int* out = a.kept + (int64_t)tgi * a.kmax;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (a.scope == FK_SCOPE_PER_FRAME && n > kRankDirect) {
    // many segments per frame (token-level rules): sort each frame in shared memory;
    // frame f's kept ids fill out[f k .. f k + k)
    unsigned long long* key = reinterpret_cast<unsigned long long*>(
        reinterpret_cast<uint8_t*>(ssc) + select_sort_off(a.max_run, n));
    int* flag = reinterpret_cast<int*>(key + select_sort_len(n));
    for (int f = 0; f < nT; ++f)
      sort_select_frame(ssc + f * n, n, a.k_frame, t_lo + f, out + f * a.k_frame, K - f * a.k_frame,
                        key, flag, warp_tot, &base_off);
    return;
  }
  if (threadIdx.x == 0) base_off = 0;
  __syncthreads();
  for (int b0 = 0; b0 < M; b0 += blockDim.x) {
    const int idx = b0 + threadIdx.x;
    bool keep = false;
    int t = 0, j = 0;
    if (idx < M) {
      t = t_lo + idx / n;
      j = idx - (idx / n) * n;
      const float* row = ssc + (idx - j);
      const float sv = row[j];
      int rank = 0;
      if (a.scope == FK_SCOPE_PER_FRAME) {
        for (int jj = 0; jj < n; ++jj) {
          const float o = row[jj];
          rank += (o < sv) || (o == sv && jj < j);
        }
        keep = rank < a.k_frame;
      } else {
        for (int qq = 0; qq < M; ++qq) {
          const float o = ssc[qq];
          rank += (o < sv) || (o == sv && qq < idx);
        }
        keep = rank < K;
      }
    }
    const unsigned mask = __ballot_sync(0xffffffffu, keep);
    if (lane == 0) warp_tot[warp] = __popc(mask);
    __syncthreads();
    int woff = base_off;
    for (int w = 0; w < warp; ++w) woff += warp_tot[w];
    const int pos = woff + __popc(mask & ((1u << lane) - 1u));
    if (keep && pos < K) out[pos] = t * n + j;   // bounded even if scores were not finite
    __syncthreads();
    if (threadIdx.x == 0) {
      int tot = 0;
      for (int w = 0; w < (int)(blockDim.x >> 5); ++w) tot += warp_tot[w];
      base_off += tot;
    }
    __syncthreads();
  }
}

// Shared-memory layout of the scoring kernel (offsets in bytes from the dynamic base).
template <int D>
struct ScoreSmem {
  static constexpr int kStageBytes = kScoreTokensPerCta * D * 2;   // one frame-chunk
  static constexpr int kBarOff = kScoreStages * kStageBytes;
  static constexpr int kAccOff = kBarOff + kScoreStages * 8;
};

// D = head_dim.  Four lanes own one token (a warp 8 tokens, the CTA the 32 tokens of one
// frame-chunk).  Lane q of a token holds channel groups g = 4*(i ^ o) + q in register slot
// i < GPL = D/32 (groups of 8 channels, 16 bytes each), o = the token's parity: with the
// odd tokens' slots swapped pairwise, the 8 lanes of each quarter-warp read 8 distinct
// 16-byte bank groups from the unswizzled staged rows.  The slot permutation i -> i ^ o is
// an automorphism of the butterfly below (it maps the pair {g, g ^ s} of every stage onto
// itself), and fp32 addition is commutative, so every slot ends with the contract value.
//
// One run: item y, segment j, token chunk c, frames k_first..k_last of the item's run, all
// owned by this CTA (it adds N(k) for each and D(k) = sum d_p(k-1, k) for k >= 1; the frame
// before k_first is loaded only as the partner of k_first).  Block-uniform arguments.
// Returns false when a wait expired (the status word records it).
template <int D>
__device__ __forceinline__ bool score_run(const ScoreArgs& a, int y, int j, int c, int k_first,
                                          int k_last, uint8_t* smem, uint32_t& seq, bool& waited) {
  using L = ScoreSmem<D>;
  constexpr int GPL = D / 32;
  const ScoreItem it = a.items[y];
  const LayerRun run = a.run[it.layer];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int q = lane & 3;
  const int tl = warp * 8 + (lane >> 2);        // token within the chunk
  const int odd = tl & 1;
  const int seg_lo = j * a.seg_len;
  const int tok0 = seg_lo + c * kScoreTokensPerCta;
  const int ntok = min(kScoreTokensPerCta, seg_lo + a.seg_len - tok0);
  const bool ok = tl < ntok;
  const int n_own = k_last - k_first + 1;
  const int k_load0 = k_first > 0 ? k_first - 1 : 0;
  const int n_load = k_last - k_load0 + 1;
  int* acc32 = reinterpret_cast<int*>(smem + L::kAccOff);   // [frame][4]: N hi, N lo, D hi, D lo
  const uint32_t sbase = su32_shared(smem);

  for (int i = threadIdx.x; i < 4 * n_own; i += blockDim.x) acc32[i] = 0;
  // producer: thread 0 streams the frame-chunks (ntok consecutive rows of a page, one
  // contiguous block) through the kScoreStages-stage ring; frame u of the run is sequence
  // number seq + u of this CTA, in stage (seq + u) % NS, phase parity ((seq + u) / NS) & 1
  const uint32_t bytes = (uint32_t)ntok * D * 2;
  const int slot_end = a.S + a.cap_nonsink;
  int next_slot = ring_slot(run.t_first + k_load0, a.S, a.cap_nonsink);
  const bf16* src0 = it.pagesK + (int64_t)tok0 * D;
  const int64_t frame_elems = (int64_t)a.F * D;
  auto issue = [&](int u) {
    // frames the previous kernel of the stream wrote (the chunk it retired) are read only
    // after that kernel has completed; older frames stream while it still runs
    if (!waited && run.t_first + k_load0 + u >= run.t_fresh) {
      pdl_wait();
      waited = true;
    }
    const uint32_t st = (seq + u) % kScoreStages;
    const uint32_t bar = sbase + L::kBarOff + st * 8;
    mbar_expect_tx(bar, bytes);
    bulk_load(sbase + st * L::kStageBytes, src0 + (int64_t)next_slot * frame_elems, bytes, bar);
    // scored frames are never sinks: the slot advances and wraps to the first non-sink slot
    next_slot = next_slot + 1 == slot_end ? a.S : next_slot + 1;
  };
  if (threadIdx.x == 0)
    for (int u = 0; u < min(kScoreStages, n_load); ++u) issue(u);

  uint4 prv[GPL];
#pragma unroll
  for (int i = 0; i < GPL; ++i) prv[i] = make_uint4(0, 0, 0, 0);   // partner of frame 0: none
  bool bad = false, timed_out = false;
  for (int u = 0; u < n_load; ++u) {
    const int k = k_load0 + u;
    const uint32_t st = (seq + u) % kScoreStages;
    if (!mbar_wait(sbase + L::kBarOff + st * 8, ((seq + u) / kScoreStages) & 1)) timed_out = true;
    uint4 cur[GPL];
    const uint32_t row = sbase + st * L::kStageBytes + tl * (D * 2) + q * 16;
#pragma unroll
    for (int i = 0; i < GPL; ++i) cur[i] = lds128(row + ((i ^ odd) * 64));
    // every thread has its registers: the stage can be refilled
    if (__syncthreads_or(timed_out)) {
      if (threadIdx.x == 0) atomicOr(a.status, kStatusTimeout);
      // drain: wait (bounded) for the copies still in flight before the CTA leaves
      for (int v = u; v < min(u + kScoreStages, n_load); ++v)
        mbar_wait(sbase + L::kBarOff + ((seq + v) % kScoreStages) * 8, ((seq + v) / kScoreStages) & 1);
      return false;
    }
    if (threadIdx.x == 0 && u + kScoreStages < n_load) issue(u + kScoreStages);
    if (k >= k_first) {
      // one fma chain per channel group (channel order), for n_p and d_p
      float nn[GPL], dd[GPL];
#pragma unroll
      for (int i = 0; i < GPL; ++i) {
        nn[i] = 0.0f;
        dd[i] = 0.0f;
        fma_word(cur[i].x, prv[i].x, nn[i], dd[i]);
        fma_word(cur[i].y, prv[i].y, nn[i], dd[i]);
        fma_word(cur[i].z, prv[i].z, nn[i], dd[i]);
        fma_word(cur[i].w, prv[i].w, nn[i], dd[i]);
      }
      // butterfly p[g] += p[g ^ s], s = D/16 .. 1: strides s >= 4 pair slot i with
      // i ^ (s/4) inside the lane, strides 2 and 1 pair lane q with q ^ s
#pragma unroll
      for (int sft = GPL / 2; sft >= 1; sft >>= 1) {
#pragma unroll
        for (int i = 0; i < GPL; ++i) {
          if ((i & sft) == 0) {
            const float n2 = __fadd_rn(nn[i], nn[i ^ sft]);
            const float d2 = __fadd_rn(dd[i], dd[i ^ sft]);
            nn[i] = n2; nn[i ^ sft] = n2;
            dd[i] = d2; dd[i ^ sft] = d2;
          }
        }
      }
#pragma unroll
      for (int sft = 2; sft >= 1; sft >>= 1) {
        nn[0] = __fadd_rn(nn[0], __shfl_xor_sync(0xffffffffu, nn[0], sft));
        dd[0] = __fadd_rn(dd[0], __shfl_xor_sync(0xffffffffu, dd[0], sft));
      }
      // lane q = 0 of a token converts n_p, lane q = 1 converts d_p (then summed over the
      // warp's tokens); the other lanes contribute zero
      int hi = 0, lo = 0;
      if (ok && q < 2) {
        const float v = q == 0 ? nn[0] : (k > 0 ? dd[0] : 0.0f);
        if (q == 0) bad |= !(nn[0] <= 8388608.0f);
        fixed24_split(v, hi, lo);
      }
#pragma unroll
      for (int sft = 4; sft < 32; sft <<= 1) {
        hi += __shfl_xor_sync(0xffffffffu, hi, sft);
        lo += __shfl_xor_sync(0xffffffffu, lo, sft);
      }
      if (lane < 2) {                            // lane 0: N(k) parts, lane 1: D(k) parts
        atomicAdd(&acc32[4 * (k - k_first) + 2 * lane], hi);
        atomicAdd(&acc32[4 * (k - k_first) + 2 * lane + 1], lo);
      }
    }
#pragma unroll
    for (int i = 0; i < GPL; ++i) prv[i] = cur[i];
  }
  seq += n_load;
  if (bad) atomicOr(a.status, kStatusRange);
  __syncthreads();
  // exact int64 adds into the target's sums (fire-and-forget; the selection kernel reads
  // them after this kernel has completed)
  unsigned long long* sums = a.sums + (int64_t)it.target * a.max_run * a.n_seg * 2;
  for (int qq = threadIdx.x; qq < 2 * n_own; qq += blockDim.x) {
    const int kk = qq >> 1, which = qq & 1;
    const long long v =
        (long long)acc32[4 * kk + 2 * which] * 16777216ll + (long long)acc32[4 * kk + 2 * which + 1];
    atomicAdd(sums + ((int64_t)(k_first + kk) * a.n_seg + j) * 2 + which, (unsigned long long)v);
  }
  __syncthreads();                               // acc32 is reused by the next run
  return true;
}

// Persistent grid: the frame-chunks of all scored items (item, segment, token chunk, frame)
// form one flattened range split into equal contiguous pieces, one per CTA; a piece walks
// its runs in order.  Launched with programmatic dependent launch after the current-chunk
// kernel: a CTA streams frames older than the retired chunk while that kernel still runs,
// waits for it (griddepcontrol.wait, thread 0, before its first fresh frame) and waits in
// any case before it exits, so this grid completes only after that kernel, and the
// selection and compaction chained behind it see the retired frames.
template <int D>
__global__ void __launch_bounds__(kScoreThreads, 4) score_kernel(const ScoreArgs a) {
  extern __shared__ __align__(128) uint8_t smem[];
  using L = ScoreSmem<D>;
  pdl_trigger();
  if (threadIdx.x == 0) {
    for (int i = 0; i < kScoreStages; ++i) mbar_init(su32_shared(smem) + L::kBarOff + i * 8, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  bool waited = false;                           // thread 0: the previous kernel has completed
  const long long T = a.total_units;
  long long g = T * blockIdx.x / gridDim.x;
  const long long g_end = T * (blockIdx.x + 1) / gridDim.x;
  const int per_item = a.n_seg * a.chunks;
  uint32_t seq = 0;
  while (g < g_end) {
    int lo = 0, hi = a.n_active - 1;             // active layer holding unit g
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (a.act_start[mid] <= g) lo = mid;
      else hi = mid - 1;
    }
    const LayerRun run = a.run[a.act_layer[lo]];
    const long long idx = g - a.act_start[lo];
    const long long chunk_id = idx / run.n_read;
    const int k = (int)(idx - chunk_id * run.n_read);
    const int item_local = (int)(chunk_id / per_item);
    const int r = (int)(chunk_id - (long long)item_local * per_item);
    const int j = r / a.chunks;
    const long long left = g_end - g;
    const int k_last = (int)(left < run.n_read - k ? k + left - 1 : run.n_read - 1);
    if (!score_run<D>(a, a.act_first_item[lo] + item_local, j, r - j * a.chunks, k, k_last, smem, seq,
                      waited))
      break;
    g += k_last - k + 1;
  }
  if (threadIdx.x == 0 && !waited) pdl_wait();
}

template <int D>
constexpr size_t score_smem_bytes_d(int max_run) {
  return (size_t)ScoreSmem<D>::kAccOff + (size_t)4 * max_run * sizeof(int);
}
size_t score_smem_bytes(int head_dim, int max_run) {
  return head_dim == 128 ? score_smem_bytes_d<128>(max_run) : score_smem_bytes_d<64>(max_run);
}
size_t select_smem_bytes(int max_run, int n_seg) {
  size_t b = (size_t)max_run * n_seg * sizeof(float);
  if (n_seg > kRankDirect)   // sort keys and flags of one frame
    b = select_sort_off(max_run, n_seg) + (size_t)select_sort_len(n_seg) * 8 + (size_t)n_seg * 4;
  return b;
}

// launch with the programmatic-dependent-launch attribute: the kernel's prologue may
// overlap the previous kernel's tail; its pdl_wait() orders it after that kernel
template <typename Kern>
cudaError_t launch_pdl(Kern kern, unsigned grid, unsigned threads, size_t smem, cudaStream_t s,
                       const ScoreArgs& a) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(threads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, a);
}

// Self-test of the bounded wait: one thread waits on an mbarrier that nothing arrives on,
// with the kernels' wait primitive and a short limit, then records the expiry in the status
// word exactly as the production kernels do and returns.
__global__ void wait_selftest_kernel(uint64_t limit_ns, int* status) {
  __shared__ __align__(8) uint64_t bar;
  const uint32_t b = su32_shared(&bar);
  mbar_init(b, 1);
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  if (!mbar_wait(b, 0, limit_ns)) atomicOr(status, kStatusTimeout);
}

}  // namespace

cudaError_t launch_wait_selftest(uint64_t limit_ns, int* status, cudaStream_t s) {
  wait_selftest_kernel<<<1, 1, 0, s>>>(limit_ns, status);
  return cudaGetLastError();
}

cudaError_t score_prepare(int head_dim, int max_run, int n_seg, int* max_ctas) {
  const int smem = (int)score_smem_bytes(head_dim, max_run);
  const void* fn = head_dim == 128 ? (const void*)score_kernel<128> : (const void*)score_kernel<64>;
  // the limits are per function and shared by every handle: only ever raise them
  cudaFuncAttributes fa{};
  cudaError_t e = cudaFuncGetAttributes(&fa, fn);
  if (e != cudaSuccess) return e;
  if (smem > 48 * 1024 && smem > fa.maxDynamicSharedSizeBytes)
    e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  const int sel_smem = (int)select_smem_bytes(max_run, n_seg);
  if ((e = cudaFuncGetAttributes(&fa, (const void*)select_kernel)) != cudaSuccess) return e;
  if (sel_smem > 48 * 1024 && sel_smem > fa.maxDynamicSharedSizeBytes)
    e = cudaFuncSetAttribute((const void*)select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             sel_smem);
  if (e != cudaSuccess) return e;
  int dev = 0, sms = 0, per_sm = 0;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
  if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, kScoreThreads, smem)) != cudaSuccess)
    return e;
  *max_ctas = sms * (per_sm > 0 ? per_sm : 1);
  return cudaSuccess;
}

void launch_score(const ScoreArgs& a, cudaStream_t s) {
  if (a.n_items == 0) return;
  const long long units = a.total_units;
  if (units <= 0) return;
  const unsigned grid = (unsigned)(units < a.max_ctas ? units : a.max_ctas);
  const size_t smem = score_smem_bytes(a.D, a.max_run);
  if (a.D == 128) launch_pdl(score_kernel<128>, grid, kScoreThreads, smem, s, a);
  else launch_pdl(score_kernel<64>, grid, kScoreThreads, smem, s, a);
}

void launch_select(const ScoreArgs& a, int n_targets, cudaStream_t s) {
  if (n_targets <= 0) return;
  if (a.rule != FK_SELECT_SIMILARITY && a.scope == FK_SCOPE_PER_FRAME && a.n_seg > kRankDirect) {
    int frames = 0;
    for (int l = 0; l < kMaxLayers; ++l) frames = std::max(frames, a.n_scoreable[l]);
    if (frames <= 0) return;
    const size_t smem = ((size_t)a.n_seg * sizeof(float) + 7) / 8 * 8 +
                        (size_t)select_sort_len(a.n_seg) * 8 + (size_t)a.n_seg * 4;
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3((unsigned)n_targets, (unsigned)frames);
    cfg.blockDim = dim3(kSelectThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cudaLaunchKernelEx(&cfg, select_frames_kernel, a);
    return;
  }
  launch_pdl(select_kernel, (unsigned)n_targets, kSelectThreads, select_smem_bytes(a.max_run, a.n_seg), s, a);
}

// ---------------------------------------------------------------------------------------
// Allocation-free scoring (fk_segment_scores_noalloc in fk.h).  The scoring kernel's scratch
// (int64 sums, a status word, its one-item tables) lives in a file-scope device array
// of fixed size instead of memory from cudaMalloc, so the call allocates nothing.  The array
// exists once per device that loads the library; every call uses it.
namespace {

constexpr int kNoAllocMaxFrames = 256;
constexpr int kNoAllocMaxSegments = 32;
constexpr int kNoAllocMaxCells = 4096;                 // n_frames * n_segments
constexpr size_t kNoAllocSumsBytes = (size_t)kNoAllocMaxCells * 2 * sizeof(unsigned long long);
constexpr size_t kNoAllocCtrOff = kNoAllocSumsBytes;   // 64-byte word block; status at +12 bytes
constexpr size_t kNoAllocItemOff = kNoAllocCtrOff + 64;
constexpr size_t kNoAllocTargetOff = kNoAllocItemOff + 64;
constexpr size_t kNoAllocBytes = kNoAllocTargetOff + 64;   // 65,728 bytes
static_assert(kNoAllocBytes == 65728, "documented size");
static_assert(sizeof(ScoreItem) <= 64 && sizeof(SelectTarget) <= 32, "table slots");

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocBytes];

struct NoAllocDevice {
  bool ready = false;
  unsigned char* scratch = nullptr;   // device address of g_noalloc_scratch on this device
  int ctas64 = 0, ctas128 = 0;        // persistent grid sizes
};
constexpr int kNoAllocMaxDevices = 64;
NoAllocDevice g_noalloc[kNoAllocMaxDevices];
std::mutex g_noalloc_mu;

bool device_pointer(const void* p) {
  cudaPointerAttributes at{};
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

// Prepares the scratch array for one call: zeroes the first n_words int64 sums and the status
// word, and writes the one-entry item table (K arrives as a kernel parameter, so no host memory
// is read) and the one-entry target table.
__global__ void noalloc_setup_kernel(unsigned char* sc, const bf16* K, int n_words) {
  unsigned long long* sums = reinterpret_cast<unsigned long long*>(sc);
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n_words; i += gridDim.x * blockDim.x)
    sums[i] = 0ull;
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    reinterpret_cast<int*>(sc + kNoAllocCtrOff)[3] = 0;
    *reinterpret_cast<ScoreItem*>(sc + kNoAllocItemOff) = ScoreItem{K, 0, 0};
    *reinterpret_cast<SelectTarget*>(sc + kNoAllocTargetOff) = SelectTarget{0, 0, 1};
  }
}

}  // namespace
}  // namespace fk

extern "C" fk_status fk_segment_scores_noalloc(const void* K, int n_frames, int tokens_per_frame,
                                                int head_dim, int n_segments, float* scores,
                                                int* status, void* stream) {
  using namespace fk;
  if (!K || !scores) return FK_ERR_ARG;
  if ((reinterpret_cast<uintptr_t>(K) & 15u) || (reinterpret_cast<uintptr_t>(scores) & 3u) ||
      (reinterpret_cast<uintptr_t>(status) & 3u))
    return FK_ERR_ARG;
  if (head_dim != 64 && head_dim != 128) return FK_ERR_CONFIG;
  if (n_segments < 1 || n_segments > kNoAllocMaxSegments) return FK_ERR_CONFIG;
  if (tokens_per_frame < 1 || tokens_per_frame % n_segments) return FK_ERR_CONFIG;
  if ((int64_t)tokens_per_frame * head_dim > (1 << 28)) return FK_ERR_CONFIG;
  if (n_frames < 2 || n_frames > kNoAllocMaxFrames || n_frames * n_segments > kNoAllocMaxCells)
    return FK_ERR_CONFIG;
  if (!device_pointer(K) || !device_pointer(scores) || (status && !device_pointer(status)))
    return FK_ERR_ARG;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kNoAllocMaxDevices) {
    cudaGetLastError();
    return FK_ERR_CUDA;
  }
  NoAllocDevice& nd = g_noalloc[dev];
  {
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    if (!nd.ready) {   // first call on this device: resolve the array's address, size the grid
      void* p = nullptr;
      if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) {
        cudaGetLastError();
        return FK_ERR_CUDA;
      }
      if (score_prepare(64, kNoAllocMaxFrames, kNoAllocMaxSegments, &nd.ctas64) != cudaSuccess ||
          score_prepare(128, kNoAllocMaxFrames, kNoAllocMaxSegments, &nd.ctas128) != cudaSuccess) {
        cudaGetLastError();
        return FK_ERR_CUDA;
      }
      nd.scratch = static_cast<unsigned char*>(p);
      nd.ready = true;
    }
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  unsigned char* sc = nd.scratch;
  // the sums and the status word must start at zero: the previous call leaves the sums
  // cleared, but the setup kernel clears them anyway (and writes the tables)
  const int n_words = n_frames * n_segments * 2;
  noalloc_setup_kernel<<<(n_words + 255) / 256, 256, 0, s>>>(sc, static_cast<const bf16*>(K), n_words);
  ScoreArgs a{};
  a.items = reinterpret_cast<const ScoreItem*>(sc + kNoAllocItemOff);
  a.targets = reinterpret_cast<const SelectTarget*>(sc + kNoAllocTargetOff);
  a.n_items = 1;
  a.F = tokens_per_frame;
  a.D = head_dim;
  a.n_seg = n_segments;
  a.seg_len = tokens_per_frame / n_segments;
  a.chunks = (a.seg_len + kScoreTokensPerCta - 1) / kScoreTokensPerCta;
  a.S = 0;                         // frames 0..n_frames-1 in slots 0..n_frames-1
  a.cap_nonsink = n_frames;
  a.ring_slots = n_frames;         // scores[t][j] for t = 0..n_frames-2
  a.max_run = n_frames;
  a.n_active = 1;
  a.act_layer[0] = 0;
  a.act_first_item[0] = 0;
  a.act_start[0] = 0;
  a.total_units = (long long)n_segments * a.chunks * n_frames;
  a.max_ctas = head_dim == 128 ? nd.ctas128 : nd.ctas64;
  a.scope = FK_SCOPE_PER_FRAME;
  a.k_frame = 0;
  a.kmax = 1;
  a.sums = reinterpret_cast<unsigned long long*>(sc);
  a.status = status ? status : reinterpret_cast<int*>(sc + kNoAllocCtrOff) + 3;
  a.scores = scores;
  a.kept = reinterpret_cast<int*>(sc + kNoAllocTargetOff + 32);   // unused: no selection
  a.run[0] = {0, n_frames, 0, n_frames};
  a.t_lo[0] = 0;
  a.n_scoreable[0] = 0;
  a.n_keep[0] = 0;
  // plain launches (no programmatic dependent launch): each kernel starts after the one
  // before it has completed, so the scoring kernel reads the tables the setup kernel wrote
  const unsigned grid = (unsigned)std::min<long long>(a.total_units, a.max_ctas);
  const size_t smem = score_smem_bytes(head_dim, a.max_run);
  if (head_dim == 128) score_kernel<128><<<grid, kScoreThreads, smem, s>>>(a);
  else score_kernel<64><<<grid, kScoreThreads, smem, s>>>(a);
  select_kernel<<<1, kSelectThreads, select_smem_bytes(a.max_run, a.n_seg), s>>>(a);
  return cudaGetLastError() == cudaSuccess ? FK_OK : FK_ERR_CUDA;
}
