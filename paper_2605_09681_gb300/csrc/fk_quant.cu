// FP8 (OCP E4M3) quantization for the FP8_QK attention (the paper's quantization appendix:
// FP8 attention on the compressed cache).  One HBM-bound streaming launch per attention call
// covers the query rows and the changed key rows:
//   queries  row r scaled by 2^-e_r, e_r the smallest integer with max |x_r| <= 448 * 2^e_r,
//            so the scaling is exact and the E4M3 rounding is the only inexact step;
//   keys     rounded unscaled (the scoring precondition |K| <= 256 keeps them inside the
//            E4M3 range; larger magnitudes saturate at 448).
// The rounding is the hardware conversion cvt.rn.satfinite.e4m3x2.f32 (to nearest, ties to
// even, saturating to the largest finite value).
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

// two floats -> two E4M3 codes, `lo` in the low byte
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

__device__ __forceinline__ float absmax8(uint4 v) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  float m = 0.0f;
#pragma unroll
  for (int i = 0; i < 4; ++i)
    m = fmaxf(m, fmaxf(fabsf(__uint_as_float(w[i] << 16)), fabsf(__uint_as_float(w[i] & 0xFFFF0000u))));
  return m;
}

// smallest e with amax <= 448 * 2^e, from the bit fields of amax (>= 0): with amax = 1.f 2^E,
// i.e. m 2^(E+1) for m = 1.f / 2 in [0.5, 1), and 448 = 0.875 * 2^9, e = E - 8 when
// m <= 0.875 (1.f <= 1.75: mantissa field <= 0x600000), else E - 7.  Subnormal amax (below
// 2^-126) and zero take the clamp / zero rule.
__device__ __forceinline__ int row_exponent(float amax) {
  const uint32_t b = __float_as_uint(amax);
  if (b == 0) return 0;
  if ((b >> 23) == 0) return -120;
  const int E = (int)(b >> 23) - 127;
  const int e = (b & 0x7FFFFFu) <= 0x600000u ? E - 8 : E - 7;
  return max(-120, min(120, e));
}

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
    const int e = row_exponent(m);
    if (g < ng) {
      dst[g] = e4m3x8(v[k], __uint_as_float((uint32_t)(127 - e) << 23));
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
