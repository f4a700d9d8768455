// FP8 (OCP E4M3) quantization for the FP8_QK attention (the paper's quantization appendix:
// FP8 attention on the compressed cache).  Both kernels are HBM-bound streaming passes: 16
// bytes of bf16 in, 8 bytes of E4M3 codes out per thread and step.
//   keys     rounded unscaled (the scoring precondition |K| <= 256 keeps them inside the
//            E4M3 range; larger magnitudes saturate at 448);
//   queries  row r scaled by 2^-e_r, e_r the smallest integer with max |x_r| <= 448 * 2^e_r,
//            so the scaling is exact and the E4M3 rounding is the only inexact step.
// The rounding is the hardware conversion cvt.rn.satfinite.e4m3x2.f32 (to nearest, ties to
// even, saturating to the largest finite value).
#include "fk_internal.h"

namespace fk {
namespace {

constexpr int kQuantThreads = 256;

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
  const int E = (int)(b >> 23) - 127;
  if ((b >> 23) == 0) return -120;
  const int e = (b & 0x7FFFFFu) <= 0x600000u ? E - 8 : E - 7;
  return max(-120, min(120, e));
}

__global__ void __launch_bounds__(kQuantThreads) quant_ranges_kernel(const QuantRanges a) {
  const int r = blockIdx.y;
  const int64_t per_row = a.D / 8;                      // granules per row
  const int64_t n = a.rows[r] * per_row;
  const int64_t g0 = a.row0[r] * per_row;
  const uint4* src = reinterpret_cast<const uint4*>(a.src) + g0;
  uint2* dst = reinterpret_cast<uint2*>(a.dst) + g0;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x)
    dst[i] = e4m3x8(__ldg(src + i), 1.0f);
}

// one row per D/8 consecutive lanes (16 lanes for D = 128, 8 for D = 64)
template <int D>
__global__ void __launch_bounds__(kQuantThreads) quant_rows_kernel(const bf16* x, int64_t rows,
                                                                     uint8_t* q8, int8_t* exps) {
  constexpr int kLanes = D / 8;
  const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t r = t / kLanes;
  const bool in = r < rows;
  const uint4 v = in ? __ldg(reinterpret_cast<const uint4*>(x) + t) : make_uint4(0, 0, 0, 0);
  float m = absmax8(v);
#pragma unroll
  for (int off = kLanes / 2; off >= 1; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
  const int e = row_exponent(m);
  if (!in) return;
  reinterpret_cast<uint2*>(q8)[t] = e4m3x8(v, __uint_as_float((uint32_t)(127 - e) << 23));
  if ((t & (kLanes - 1)) == 0) exps[r] = (int8_t)e;
}

}  // namespace

void launch_quant_ranges(const QuantRanges& a, cudaStream_t s) {
  int64_t most = 0;
  for (int i = 0; i < a.n; ++i) most = a.rows[i] > most ? a.rows[i] : most;
  if (a.n <= 0 || most <= 0) return;
  const int64_t granules = most * (a.D / 8);
  const int64_t blocks = (granules + kQuantThreads - 1) / kQuantThreads;
  const unsigned gx = (unsigned)(blocks < 4096 ? blocks : 4096);
  quant_ranges_kernel<<<dim3(gx, (unsigned)a.n), kQuantThreads, 0, s>>>(a);
}

void launch_quant_rows_scaled(const bf16* x, int64_t rows, int D, uint8_t* q8, int8_t* exps,
                              cudaStream_t s) {
  if (rows <= 0) return;
  const int64_t threads = rows * (D / 8);
  const unsigned grid = (unsigned)((threads + kQuantThreads - 1) / kQuantThreads);
  if (D == 128) quant_rows_kernel<128><<<grid, kQuantThreads, 0, s>>>(x, rows, q8, exps);
  else quant_rows_kernel<64><<<grid, kQuantThreads, 0, s>>>(x, rows, q8, exps);
}

}  // namespace fk
