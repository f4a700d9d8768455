// Segment-wise similarity scoring and BottomK selection (Sec. 4.3, Eq. 3) in one launch.
//
// Each CTA owns a few tokens of one segment of one scored (layer, head) and streams that
// token range through the run of consecutive history frames, 16 bytes per lane, with a
// four-frame register prefetch ring; every key byte is read once.  Per token it forms the
// score-contract quantities (fp32 channel dot in a fixed fma/butterfly order, scaled by 2^24
// and truncated to int64, carried as two exact int32 halves): the squared norm n_p(t) and
// the dot d_p(t-1, t).  Warp sums go into shared-memory int32 accumulators (at most 32
// tokens per CTA, so no overflow) and each CTA adds them as int64 into the target's global
// int64 sums (exact integer adds, so the order is free).  The last CTA of a selection
// target (counted with a global atomic)
// finishes s = D / sqrt(N_t N_{t+1}) in IEEE double, stores the fp32 scores per frame slot,
// ranks the scoreable candidates by (score, segment id) and stream-compacts the kept
// segment ids with warp ballots and prefix sums.
#include <mutex>

#include "fk_internal.h"

namespace fk {
namespace {

__device__ __forceinline__ uint4 ld_keys(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
  return v;
}

// Two channels (one 32-bit word: low half first) of the norm and dot fma chains, with the
// bf16 values used directly as fma operands (fp32 product and accumulation, one rounding):
// n += c*c and d += p*c for the low channel, then for the high channel.
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

__device__ __forceinline__ int ring_slot(int f, int S, int cap) {
  return f < S ? f : S + (f - S) % cap;
}

__device__ __forceinline__ float finish_score(long long dsum, long long n1, long long n2) {
  if (n1 == 0 || n2 == 0) return 0.0f;
  const double den = __dsqrt_rn(__dmul_rn(__ll2double_rn(n1), __ll2double_rn(n2)));
  return __double2float_rn(__ddiv_rn(__ll2double_rn(dsum), den));
}

// Finish the scored pairs of target `tgi` and select its kept segments (one CTA).
__device__ void finish_and_select(const ScoreArgs& a, int tgi, int* stage) {
  __shared__ int warp_tot[32];
  __shared__ int base_off;
  const SelectTarget tg = a.targets[tgi];
  const int l = tg.layer;
  const LayerRun run = a.run[l];
  const int n = a.n_seg;
  float* sc = a.scores + (int64_t)tgi * a.ring_slots * n;

  // 1. finish the pairs (t, t+1) scored by this launch from the target's int64 sums
  //    (read past L1: other CTAs added them), then clear the sums for the next launch
  unsigned long long* sums = a.sums + (int64_t)tgi * a.max_run * n * 2;
  if (run.n_run >= 2) {
    const int pairs = (run.n_run - 1) * n;
    for (int idx = threadIdx.x; idx < pairs; idx += blockDim.x) {
      const int k = idx / n, j = idx - k * n;
      const unsigned long long N1 = __ldcg(sums + ((int64_t)k * n + j) * 2);
      const unsigned long long N2 = __ldcg(sums + ((int64_t)(k + 1) * n + j) * 2);
      const unsigned long long Dd = __ldcg(sums + ((int64_t)(k + 1) * n + j) * 2 + 1);
      const int slot = ring_slot(run.t_first + k, a.S, a.cap_nonsink);
      sc[slot * n + j] = finish_score((long long)Dd, (long long)N1, (long long)N2);
    }
  }
  __syncthreads();
  for (int i = threadIdx.x; i < run.n_run * n * 2; i += blockDim.x) sums[i] = 0ull;

  // 2. BottomK over the scoreable frames, compacted in ascending segment-id order; the
  //    window's scores are staged in shared memory in candidate order (t - t_lo)*n + j
  const int nT = a.n_scoreable[l];
  const int M = nT * n;
  const int K = a.n_keep[l];
  const int t_lo = a.t_lo[l];
  int* out = a.kept + (int64_t)tgi * a.kmax;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float* ssc = reinterpret_cast<float*>(stage);
  for (int idx = threadIdx.x; idx < M; idx += blockDim.x) {
    const int t = t_lo + idx / n, jj = idx - (idx / n) * n;
    ssc[idx] = __ldcg(sc + ring_slot(t, a.S, a.cap_nonsink) * n + jj);
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
      const float s = row[j];
      int rank = 0;
      if (a.scope == FK_SCOPE_PER_FRAME) {
        for (int jj = 0; jj < n; ++jj) {
          const float o = row[jj];
          rank += (o < s) || (o == s && jj < j);
        }
        keep = rank < a.k_frame;
      } else {
        for (int qq = 0; qq < M; ++qq) {
          const float o = ssc[qq];
          rank += (o < s) || (o == s && qq < idx);
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

// D = head_dim.  Four lanes own one token: lane q of the token holds channel groups
// 4i + q, i < GPL (GPL = D/32 groups of 8 channels, one 16-byte granule each), so each
// load instruction reads 64 contiguous bytes per token; a warp covers 8 tokens and a
// 128-thread CTA 32 tokens of one segment.
// One work unit: item y, segment j, token chunk c, sub-run z (block-uniform arguments).
template <int D>
__device__ __forceinline__ void score_unit(const ScoreArgs& a, int y, int j, int c, int z,
                                           int* acc32, int& is_last) {
  constexpr int LPT = 4;                       // lanes per token
  constexpr int GPL = D / 32;                  // granules (channel groups) per lane
  constexpr int TPW = 32 / LPT;                // tokens per warp
  constexpr int TB = (kScoreThreads / 32) * TPW;
  constexpr int PF = 4;                        // ring of packed frames per lane
  const ScoreItem it = a.items[y];
  const LayerRun run = a.run[it.layer];
  // sub-run blockIdx.z: frames k_lo .. k_hi of the run (pairs (k-1, k) for k_lo < k <= k_hi);
  // a sub-run's first frame is the previous sub-run's last one, whose norm that one counts
  const int n_sub = run.n_run > 1 ? (run.n_run - 2) / kScorePairsPerCta + 1 : 1;
  if (run.n_run == 0 || z >= n_sub) return;
  const int k_lo = z * kScorePairsPerCta;
  const int k_hi = min(k_lo + kScorePairsPerCta, run.n_run - 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int seg_lo = j * a.seg_len;
  const int tok0 = seg_lo + c * TB;
  const int tok_end = min(tok0 + TB, seg_lo + a.seg_len);
  const int q = lane % LPT;                    // lane within the token
  const int tok = tok0 + warp * TPW + lane / LPT;
  const bool ok = tok < tok_end;

  for (int i = threadIdx.x; i < 4 * run.n_run; i += blockDim.x) acc32[i] = 0;
  __syncthreads();

  const bf16* base = it.pagesK + (int64_t)tok * D + q * 8;
  const int64_t frame_elems = (int64_t)a.F * D;
  // ring slot of the next frame to load; scored frames are never sinks, so the slot
  // advances by one and wraps from the last slot to the first non-sink slot
  const int slot_end = a.S + a.cap_nonsink;
  int next_slot = ring_slot(run.t_first + k_lo, a.S, a.cap_nonsink);
  auto load = [&](int k, uint4 (&dst)[GPL]) {
#pragma unroll
    for (int i = 0; i < GPL; ++i) dst[i] = make_uint4(0, 0, 0, 0);
    if (k <= k_hi) {
      if (ok) {
        const bf16* p = base + (int64_t)next_slot * frame_elems;
#pragma unroll
        for (int i = 0; i < GPL; ++i) dst[i] = ld_keys(p + i * 32);
      }
      next_slot = next_slot + 1 == slot_end ? a.S : next_slot + 1;
    }
  };
  // ring of PF packed frames: frame k lives in buf[(k - k_lo) % PF]; the previous frame is
  // the previous slot, and a slot is refilled (PF - 1 frames ahead) once it has served as
  // "previous"
  uint4 buf[PF][GPL];
#pragma unroll
  for (int u = 0; u < PF - 1; ++u) load(k_lo + u, buf[u]);
#pragma unroll
  for (int i = 0; i < GPL; ++i) buf[PF - 1][i] = make_uint4(0, 0, 0, 0);   // "previous" of k_lo
  bool bad = false;
  for (int k0 = k_lo; k0 <= k_hi; k0 += PF) {
#pragma unroll
    for (int u = 0; u < PF; ++u) {
      const int k = k0 + u;
      if (k > k_hi) break;
      const uint4 (&cur)[GPL] = buf[u];
      const uint4 (&prv)[GPL] = buf[(u + PF - 1) % PF];
      // one fma chain per channel group (channel order), for n_p and d_p
      float n[GPL], d[GPL];
#pragma unroll
      for (int i = 0; i < GPL; ++i) {
        n[i] = 0.0f;
        d[i] = 0.0f;
        fma_word(cur[i].x, prv[i].x, n[i], d[i]);
        fma_word(cur[i].y, prv[i].y, n[i], d[i]);
        fma_word(cur[i].z, prv[i].z, n[i], d[i]);
        fma_word(cur[i].w, prv[i].w, n[i], d[i]);
      }
      load(k + PF - 1, buf[(u + PF - 1) % PF]);   // the previous frame's slot is free now
      // butterfly p[g] += p[g ^ s], s = D/16 .. 1 over groups g = 4i + q: strides s >= 4 pair
      // i with i ^ (s/4) inside the lane, strides 2 and 1 pair lane q with q ^ s
#pragma unroll
      for (int sft = GPL / 2; sft >= 1; sft >>= 1) {
#pragma unroll
        for (int i = 0; i < GPL; ++i) {
          if ((i & sft) == 0) {
            const float nn = __fadd_rn(n[i], n[i ^ sft]);
            const float dd = __fadd_rn(d[i], d[i ^ sft]);
            n[i] = nn; n[i ^ sft] = nn;
            d[i] = dd; d[i ^ sft] = dd;
          }
        }
      }
#pragma unroll
      for (int sft = 2; sft >= 1; sft >>= 1) {
        n[0] = __fadd_rn(n[0], __shfl_xor_sync(0xffffffffu, n[0], sft));
        d[0] = __fadd_rn(d[0], __shfl_xor_sync(0xffffffffu, d[0], sft));
      }
      const float np = n[0];
      const float dp = d[0];                     // 0 for the first frame of the run
      // lane q = 0 of a token converts n_p, lane q = 1 converts d_p (then summed over the
      // warp's tokens); the other lanes contribute zero
      // the norm of a sub-run's last frame belongs to the next sub-run (except at the end)
      const bool count_n = k < k_hi || k_hi == run.n_run - 1;
      int hi = 0, lo = 0;
      if (ok && q < 2) {
        const float v = q == 0 ? (count_n ? np : 0.0f) : (k > k_lo ? dp : 0.0f);
        if (q == 0) bad |= !(np <= 8388608.0f);
        fixed24_split(v, hi, lo);
      }
#pragma unroll
      for (int sft = LPT; sft < 32; sft <<= 1) {
        hi += __shfl_xor_sync(0xffffffffu, hi, sft);
        lo += __shfl_xor_sync(0xffffffffu, lo, sft);
      }
      if (lane < 2) {                            // lane 0: N(t) parts, lane 1: D(t-1, t) parts
        atomicAdd(&acc32[4 * k + 2 * lane], hi);
        atomicAdd(&acc32[4 * k + 2 * lane + 1], lo);
      }
    }
  }
  if (bad) atomicOr(a.status, kStatusRange);
  __syncthreads();
  unsigned long long* sums = a.sums + (int64_t)it.target * a.max_run * a.n_seg * 2;
  for (int qq = 2 * k_lo + threadIdx.x; qq < 2 * (k_hi + 1); qq += blockDim.x) {
    const int k = qq >> 1, which = qq & 1;
    const long long v = (long long)acc32[4 * k + 2 * which] * 16777216ll + (long long)acc32[4 * k + 2 * which + 1];
    atomicAdd(sums + ((int64_t)k * a.n_seg + j) * 2 + which, (unsigned long long)v);
  }

  // the last CTA of this item's selection target finishes it
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) {
    const SelectTarget tg = a.targets[it.target];
    const int expected = a.n_seg * a.chunks * tg.n_items * n_sub;
    is_last = atomicAdd(&a.counters[it.target], 1) == expected - 1;
  }
  __syncthreads();
  if (!is_last) return;
  __threadfence();
  finish_and_select(a, it.target, acc32);
  if (threadIdx.x == 0) a.counters[it.target] = 0;
  __syncthreads();                               // acc32 is reused by the next unit
}

// Persistent grid (one wave): CTAs take work units from a global counter until none is left;
// the last CTA to leave resets the counter for the next launch.
template <int D>
__global__ void __launch_bounds__(kScoreThreads, 4) score_kernel(const ScoreArgs a) {
  extern __shared__ int acc32[];               // [n_run][4] : {N hi, N lo, D hi, D lo}
  __shared__ int s_unit, is_last;
  const int per_sub = a.n_seg * a.chunks;
  const int per_item = per_sub * a.n_sub_max;
  const int total = a.n_items * per_item;
  for (;;) {
    if (threadIdx.x == 0) s_unit = atomicAdd(a.work, 1);
    __syncthreads();
    const int unit = s_unit;
    __syncthreads();
    if (unit >= total) break;
    const int y = unit / per_item;
    const int r = unit - y * per_item;
    const int z = r / per_sub;
    const int r2 = r - z * per_sub;
    const int j = r2 / a.chunks;
    score_unit<D>(a, y, j, r2 - j * a.chunks, z, acc32, is_last);
  }
  if (threadIdx.x == 0) {
    __threadfence();
    if (atomicAdd(a.work + 1, 1) == (int)gridDim.x - 1) {
      a.work[0] = 0;
      a.work[1] = 0;
    }
  }
}

}  // namespace

cudaError_t score_prepare(int head_dim, int max_run, int n_seg, int* max_ctas) {
  const int smem = score_smem_ints(max_run, n_seg) * (int)sizeof(int);
  const void* fn = head_dim == 128 ? (const void*)score_kernel<128> : (const void*)score_kernel<64>;
  cudaError_t e = cudaSuccess;
  if (smem > 48 * 1024) e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
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
  const int64_t units = (int64_t)a.n_items * a.n_seg * a.chunks * a.n_sub_max;
  const unsigned grid = (unsigned)(units < a.max_ctas ? units : a.max_ctas);
  const size_t smem = (size_t)score_smem_ints(a.max_run, a.n_seg) * sizeof(int);
  if (a.D == 128) score_kernel<128><<<grid, kScoreThreads, smem, s>>>(a);
  else score_kernel<64><<<grid, kScoreThreads, smem, s>>>(a);
}

// ---------------------------------------------------------------------------------------
// Allocation-free scoring (fk_segment_scores_noalloc in fk.h).  The scoring kernel's scratch
// (int64 sums, CTA and work counters, its one-item tables) lives in a file-scope device array
// of fixed size instead of memory from cudaMalloc, so the call allocates nothing.  The array
// exists once per device that loads the library; every call uses it.
namespace {

constexpr int kNoAllocMaxFrames = 256;
constexpr int kNoAllocMaxSegments = 32;
constexpr int kNoAllocMaxCells = 4096;                 // n_frames * n_segments
constexpr size_t kNoAllocSumsBytes = (size_t)kNoAllocMaxCells * 2 * sizeof(unsigned long long);
constexpr size_t kNoAllocCtrOff = kNoAllocSumsBytes;   // target counter, work[2], status
constexpr size_t kNoAllocItemOff = kNoAllocCtrOff + 64;
constexpr size_t kNoAllocTargetOff = kNoAllocItemOff + 64;
constexpr size_t kNoAllocBytes = kNoAllocTargetOff + 64;   // 65,728 bytes
static_assert(kNoAllocBytes == 65728, "documented size");

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

}  // namespace
}  // namespace fk

extern "C" fk_status fk_segment_scores_noalloc(const void* K, int n_frames, int tokens_per_frame,
                                                int head_dim, int n_segments, float* scores,
                                                void* stream) {
  using namespace fk;
  if (!K || !scores) return FK_ERR_ARG;
  if ((reinterpret_cast<uintptr_t>(K) & 15u) || (reinterpret_cast<uintptr_t>(scores) & 3u))
    return FK_ERR_ARG;
  if (head_dim != 64 && head_dim != 128) return FK_ERR_CONFIG;
  if (n_segments < 1 || n_segments > kNoAllocMaxSegments) return FK_ERR_CONFIG;
  if (tokens_per_frame < 1 || tokens_per_frame % n_segments) return FK_ERR_CONFIG;
  if ((int64_t)tokens_per_frame * head_dim > (1 << 28)) return FK_ERR_CONFIG;
  if (n_frames < 2 || n_frames > kNoAllocMaxFrames || n_frames * n_segments > kNoAllocMaxCells)
    return FK_ERR_CONFIG;
  if (!device_pointer(K) || !device_pointer(scores)) return FK_ERR_ARG;
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
  // the sums and counters must start at zero; the previous call leaves them cleared, but
  // clear them here anyway
  const size_t sums_bytes = (size_t)n_frames * n_segments * 2 * sizeof(unsigned long long);
  if (cudaMemsetAsync(sc, 0, sums_bytes, s) != cudaSuccess ||
      cudaMemsetAsync(sc + kNoAllocCtrOff, 0, 64, s) != cudaSuccess) {
    cudaGetLastError();
    return FK_ERR_CUDA;
  }
  const ScoreItem item{static_cast<const bf16*>(K), 0, 0};
  const SelectTarget target{0, 0, 1};
  if (cudaMemcpyAsync(sc + kNoAllocItemOff, &item, sizeof(item), cudaMemcpyHostToDevice, s) != cudaSuccess ||
      cudaMemcpyAsync(sc + kNoAllocTargetOff, &target, sizeof(target), cudaMemcpyHostToDevice, s) !=
          cudaSuccess) {
    cudaGetLastError();
    return FK_ERR_CUDA;
  }
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
  a.max_active_run = n_frames;
  a.n_sub_max = (n_frames - 2) / kScorePairsPerCta + 1;
  a.max_ctas = head_dim == 128 ? nd.ctas128 : nd.ctas64;
  a.scope = FK_SCOPE_PER_FRAME;
  a.k_frame = 0;
  a.kmax = 1;
  a.sums = reinterpret_cast<unsigned long long*>(sc);
  a.counters = reinterpret_cast<int*>(sc + kNoAllocCtrOff);
  a.work = reinterpret_cast<int*>(sc + kNoAllocCtrOff) + 1;
  a.status = reinterpret_cast<int*>(sc + kNoAllocCtrOff) + 3;
  a.scores = scores;
  a.kept = reinterpret_cast<int*>(sc + kNoAllocTargetOff + 32);   // unused: no selection
  a.run[0] = {0, n_frames};
  a.t_lo[0] = 0;
  a.n_scoreable[0] = 0;
  a.n_keep[0] = 0;
  launch_score(a, s);
  return cudaGetLastError() == cudaSuccess ? FK_OK : FK_ERR_CUDA;
}
