// Segment-wise similarity scoring and BottomK selection (Sec. 4.3, Eq. 3).
//
// score_kernel streams the key pages of a run of consecutive history frames once,
// 16 bytes per lane, and produces per CTA the int64 sums N_t = sum_p n_p(t) and
// D_t = sum_p d_p(t-1, t) over its tokens of one segment (the score contract: per
// token fp32 dot in a fixed fma/butterfly order, scaled by 2^24 and truncated to
// int64, so that the cross-token and cross-CTA sums are exact and order-free).
// select_kernel finishes s = D / sqrt(N_t N_{t+1}) in IEEE double, stores the fp32
// score per frame slot, ranks the scoreable candidates by (score, segment id) and
// stream-compacts the kept segment ids with warp ballots and prefix sums.
#include "fk_internal.h"

namespace fk {
namespace {

__device__ __forceinline__ uint4 ld_keys(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
  return v;
}

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

// fp32 fma chain over the 8 channels of one 16-byte granule, channel order = memory order
__device__ __forceinline__ float dot8(const uint4 a, const uint4 b) {
  float acc = 0.0f;
  acc = __fmaf_rn(bf_lo(a.x), bf_lo(b.x), acc);
  acc = __fmaf_rn(bf_hi(a.x), bf_hi(b.x), acc);
  acc = __fmaf_rn(bf_lo(a.y), bf_lo(b.y), acc);
  acc = __fmaf_rn(bf_hi(a.y), bf_hi(b.y), acc);
  acc = __fmaf_rn(bf_lo(a.z), bf_lo(b.z), acc);
  acc = __fmaf_rn(bf_hi(a.z), bf_hi(b.z), acc);
  acc = __fmaf_rn(bf_lo(a.w), bf_lo(b.w), acc);
  acc = __fmaf_rn(bf_hi(a.w), bf_hi(b.w), acc);
  return acc;
}

// butterfly over the LPT lanes that own one token: p[g] += p[g ^ s], s = LPT/2 .. 1
template <int LPT>
__device__ __forceinline__ float token_reduce(float v) {
#pragma unroll
  for (int s = LPT / 2; s >= 1; s >>= 1) v = __fadd_rn(v, __shfl_xor_sync(0xffffffffu, v, s));
  return v;
}

__device__ __forceinline__ unsigned long long fixed24(float v) {
  return (unsigned long long)__float2ll_rz(__fmul_rn(v, 16777216.0f));
}

__device__ __forceinline__ unsigned long long warp_sum_u64(unsigned long long v) {
#pragma unroll
  for (int s = 16; s >= 1; s >>= 1) v += __shfl_xor_sync(0xffffffffu, v, s);
  return v;
}

__device__ __forceinline__ int ring_slot(int f, int S, int cap) {
  return f < S ? f : S + (f - S) % cap;
}

// D = head_dim; LPT = lanes per token (one 16-byte granule each)
template <int D>
__global__ void __launch_bounds__(256) score_kernel(const ScoreArgs a) {
  constexpr int LPT = D / 8;
  constexpr int TPW = 32 / LPT;                // tokens per warp per pass
  constexpr int TPP = 8 * TPW;                 // tokens per CTA per pass
  constexpr int PASSES = kScoreTokens / TPP;   // passes per frame
  static_assert(PASSES >= 1 && kScoreTokens % TPP == 0, "token tiling");
  __shared__ unsigned long long red[8][2];

  const ScoreItem it = a.items[blockIdx.y];
  const LayerRun run = a.run[it.layer];
  if (run.n_run == 0) return;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int j = blockIdx.x / a.chunks;
  const int c = blockIdx.x - j * a.chunks;
  const int seg_lo = j * a.seg_len;
  const int tok0 = seg_lo + c * kScoreTokens;
  const int tok_end = min(tok0 + kScoreTokens, seg_lo + a.seg_len);
  const int g = lane % LPT;
  const int sub = lane / LPT;

  int tok[PASSES];
  bool ok[PASSES];
#pragma unroll
  for (int p = 0; p < PASSES; ++p) {
    tok[p] = tok0 + p * TPP + warp * TPW + sub;
    ok[p] = tok[p] < tok_end;
  }

  uint4 prev[PASSES], cur[PASSES];
  const uint4 zero = make_uint4(0, 0, 0, 0);
  auto load_frame = [&](int k, uint4 (&dst)[PASSES]) {
    const int slot = ring_slot(run.t_first + k, a.S, a.cap_nonsink);
    const bf16* base = it.pagesK + (int64_t)slot * a.F * D;
#pragma unroll
    for (int p = 0; p < PASSES; ++p)
      dst[p] = ok[p] ? ld_keys(base + (int64_t)tok[p] * D + g * 8) : zero;
  };

  load_frame(0, cur);
  for (int k = 0; k < run.n_run; ++k) {
    uint4 nxt[PASSES];
    if (k + 1 < run.n_run) load_frame(k + 1, nxt);   // one frame of prefetch
    unsigned long long accN = 0, accD = 0;
    bool bad = false;
#pragma unroll
    for (int p = 0; p < PASSES; ++p) {
      const float np = token_reduce<LPT>(dot8(cur[p], cur[p]));
      float dp = 0.0f;
      if (k > 0) dp = token_reduce<LPT>(dot8(prev[p], cur[p]));
      if (g == 0 && ok[p]) {
        bad |= !(np <= 8388608.0f);
        accN += fixed24(np);
        accD += fixed24(dp);
      }
    }
    if (bad) atomicOr(a.status, kStatusRange);
    accN = warp_sum_u64(accN);
    accD = warp_sum_u64(accD);
    if (lane == 0) { red[warp][0] = accN; red[warp][1] = accD; }
    __syncthreads();
    if (threadIdx.x == 0) {
      unsigned long long sN = 0, sD = 0;
#pragma unroll
      for (int w = 0; w < 8; ++w) { sN += red[w][0]; sD += red[w][1]; }
      const int64_t idx =
          (((int64_t)blockIdx.y * a.max_run + k) * a.n_seg + j) * a.chunks + c;
      reinterpret_cast<longlong2*>(a.partials)[idx] = make_longlong2((long long)sN, (long long)sD);
    }
    __syncthreads();
#pragma unroll
    for (int p = 0; p < PASSES; ++p) { prev[p] = cur[p]; if (k + 1 < run.n_run) cur[p] = nxt[p]; }
  }
}

__device__ __forceinline__ float finish_score(long long dsum, long long n1, long long n2) {
  if (n1 == 0 || n2 == 0) return 0.0f;
  const double den = __dsqrt_rn(__dmul_rn(__ll2double_rn(n1), __ll2double_rn(n2)));
  return __double2float_rn(__ddiv_rn(__ll2double_rn(dsum), den));
}

// one CTA per selection target
__global__ void __launch_bounds__(256) select_kernel(const SelectArgs a) {
  __shared__ int warp_tot[8];
  __shared__ int base_off;
  const SelectTarget tg = a.targets[blockIdx.x];
  const int l = tg.layer;
  const LayerRun run = a.run[l];
  const int n = a.n_seg;
  float* sc = a.scores + (int64_t)blockIdx.x * a.ring_slots * n;

  // 1. finish the pairs (t, t+1) scored by this launch
  if (run.n_run >= 2) {
    const int pairs = (run.n_run - 1) * n;
    for (int idx = threadIdx.x; idx < pairs; idx += blockDim.x) {
      const int k = idx / n, j = idx - k * n;
      long long N1 = 0, N2 = 0, Dd = 0;
      for (int i = 0; i < tg.n_items; ++i) {
        const longlong2* P = reinterpret_cast<const longlong2*>(a.partials) +
                             ((int64_t)(tg.first_item + i) * a.max_run) * n * a.chunks;
        for (int c = 0; c < a.chunks; ++c) {
          const longlong2 x = P[((int64_t)k * n + j) * a.chunks + c];
          const longlong2 y = P[((int64_t)(k + 1) * n + j) * a.chunks + c];
          N1 += x.x;
          N2 += y.x;
          Dd += y.y;
        }
      }
      const int slot = ring_slot(run.t_first + k, a.S, a.cap_nonsink);
      sc[slot * n + j] = finish_score(Dd, N1, N2);
    }
  }
  __syncthreads();

  // 2. BottomK over the scoreable frames, compacted in ascending segment-id order
  const int nT = a.n_scoreable[l];
  const int M = nT * n;
  const int K = a.n_keep[l];
  const int t_lo = a.t_lo[l];
  int* out = a.kept + (int64_t)blockIdx.x * a.kmax;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) base_off = 0;
  __syncthreads();
  for (int b0 = 0; b0 < M; b0 += blockDim.x) {
    const int idx = b0 + threadIdx.x;
    bool keep = false;
    int t = 0, j = 0;
    if (idx < M) {
      t = t_lo + idx / n;
      j = idx - (idx / n) * n;
      const float s = sc[ring_slot(t, a.S, a.cap_nonsink) * n + j];
      int rank = 0;
      if (a.scope == FK_SCOPE_PER_FRAME) {
        const float* row = sc + ring_slot(t, a.S, a.cap_nonsink) * n;
        for (int jj = 0; jj < n; ++jj) {
          const float o = row[jj];
          rank += (o < s) || (o == s && jj < j);
        }
        keep = rank < a.k_frame;
      } else {
        for (int q = 0; q < M; ++q) {
          const int tq = t_lo + q / n, jq = q - (q / n) * n;
          const float o = sc[ring_slot(tq, a.S, a.cap_nonsink) * n + jq];
          rank += (o < s) || (o == s && q < idx);
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
      for (int w = 0; w < 8; ++w) tot += warp_tot[w];
      base_off += tot;
    }
    __syncthreads();
  }
}

}  // namespace

void launch_score(const ScoreArgs& a, cudaStream_t s) {
  if (a.n_items == 0) return;
  dim3 grid((unsigned)(a.n_seg * a.chunks), (unsigned)a.n_items);
  if (a.D == 128) score_kernel<128><<<grid, 256, 0, s>>>(a);
  else score_kernel<64><<<grid, 256, 0, s>>>(a);
}

void launch_select(const SelectArgs& a, cudaStream_t s) {
  if (a.n_targets == 0) return;
  select_kernel<<<(unsigned)a.n_targets, 256, 0, s>>>(a);
}

}  // namespace fk
