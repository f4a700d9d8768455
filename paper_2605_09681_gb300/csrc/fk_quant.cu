// FP8 (OCP E4M3) quantization for the FP8_QK attention (the paper's quantization appendix:
// FP8 attention on the compressed cache): one HBM-bound streaming launch over query rows and /
// or key row ranges:
//   queries  row r scaled by 2^-e_r, e_r the smallest integer with max |x_r| <= 448 * 2^e_r,
//            so the scaling is exact and the E4M3 rounding is the only inexact step;
//   keys     rounded unscaled (E4M3's relative precision is the same across its normal
//            range 2^-6..448; key elements beyond 448 saturate, so FP8_QK requires keys
//            within +-448).
// The rounding is the hardware conversion cvt.rn.satfinite.e4m3x2.f32 (to nearest, ties to
// even, saturating to the largest finite value) and the exponent rule is e4m3_row_exponent,
// both in fk_internal.h and shared with the attention kernel, which quantizes its own query
// tiles; the views' E4M3 keys are written by the copy kernels (fk_copy.cu).  This launch
// serves fk_quantize_e4m3.
// Work split: every part (the queries, each key range) is cut into chunks of kQuantChunk
// 16-byte granules of bf16, one chunk per block; thread t converts granules t, t + 256,
// t + 512 and t + 768 of its chunk, with all four loads issued before the first conversion
// (64 bytes in flight per thread).  Chunks start at multiples of 1024 granules, so the D/8
// lanes holding one query row are always consecutive lanes of one warp.
#include "fk_internal.h"

namespace fk {
namespace {

constexpr int kQuantThreads = 256;
constexpr int kQuantUnroll = 4;
constexpr int kQuantChunk = kQuantThreads * kQuantUnroll;

template <int LANES>   // lanes per query row: D / 8
__device__ __forceinline__ void quant_query_chunk(const QuantArgs& a, int64_t c0) {
  const int64_t ng = a.q_rows * LANES;
  const uint4* src = reinterpret_cast<const uint4*>(a.q_src);
  uint2* dst = reinterpret_cast<uint2*>(a.q_dst);
  uint4 v[kQuantUnroll];
#pragma unroll
  for (int k = 0; k < kQuantUnroll; ++k) {
    const int64_t g = c0 + k * kQuantThreads + threadIdx.x;
    v[k] = g < ng ? __ldg(src + g) : make_uint4(0, 0, 0, 0);
  }
#pragma unroll
  for (int k = 0; k < kQuantUnroll; ++k) {
    const int64_t g = c0 + k * kQuantThreads + threadIdx.x;
    float m = absmax8(v[k]);
#pragma unroll
    for (int off = LANES / 2; off >= 1; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
    const int e = e4m3_row_exponent(m);
    if (g < ng) {
      dst[g] = e4m3x8(v[k], pow2f(-e));
      if ((threadIdx.x & (LANES - 1)) == 0) a.q_exp[g / LANES] = (int8_t)e;
    }
  }
}

__global__ void __launch_bounds__(kQuantThreads) quant_kernel(const QuantArgs a) {
  const int64_t b = blockIdx.x;
  int lo = 0, hi = a.n;                          // part p: blk[p] <= b < blk[p + 1]
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (a.blk[mid] <= b) lo = mid;
    else hi = mid - 1;
  }
  const int64_t c0 = (b - a.blk[lo]) * kQuantChunk;
  if (lo == 0) {                                 // query rows
    if (a.q_dim == 128) quant_query_chunk<16>(a, c0);
    else quant_query_chunk<8>(a, c0);
    return;
  }
  const int r = lo - 1;                          // key range r
  const int64_t per_row = a.k_dim / 8;
  const int64_t ng = a.rows[r] * per_row;
  const int64_t g0 = a.row0[r] * per_row;
  const uint4* src = reinterpret_cast<const uint4*>(a.k_src) + g0;
  uint2* dst = reinterpret_cast<uint2*>(a.k_dst) + g0;
  uint4 v[kQuantUnroll];
#pragma unroll
  for (int k = 0; k < kQuantUnroll; ++k) {
    const int64_t g = c0 + k * kQuantThreads + threadIdx.x;
    if (g < ng) v[k] = __ldg(src + g);
  }
#pragma unroll
  for (int k = 0; k < kQuantUnroll; ++k) {
    const int64_t g = c0 + k * kQuantThreads + threadIdx.x;
    if (g < ng) dst[g] = e4m3x8(v[k], 1.0f);
  }
}

}  // namespace

void launch_quant(QuantArgs& a, cudaStream_t s) {
  const auto blocks = [](int64_t granules) { return (granules + kQuantChunk - 1) / kQuantChunk; };
  a.blk[0] = 0;
  a.blk[1] = a.q_rows > 0 ? blocks(a.q_rows * (a.q_dim / 8)) : 0;
  for (int i = 0; i < a.n; ++i) a.blk[i + 2] = a.blk[i + 1] + blocks(a.rows[i] * (a.k_dim / 8));
  const int64_t total = a.blk[a.n + 1];
  if (total <= 0) return;
  quant_kernel<<<(unsigned)total, kQuantThreads, 0, s>>>(a);
}

}  // namespace fk
