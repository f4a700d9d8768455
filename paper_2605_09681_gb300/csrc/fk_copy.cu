// Data-movement kernels of the Forcing-KV cache: the current-chunk update (the previous
// current chunk joins the history pages, and the views' sink and anchor slots where it holds
// those frames, and the new chunk is scattered from the caller's token-major [tokens][H][D]
// layout into the per-head views, in one pass; it can also form the scoring sums of the frames
// it retires), the prefill scatter of history frames, and the gather of kept segments into the
// packed per-head views of dynamic heads (Sec. 4.3, Eq. 4: sink, kept segments and the anchor
// frame; attention does not depend on the order of the keys, so a view holds them as
// [current chunk | sinks | anchor | kept-segment ring] and incremental compaction only appends).
// All of them are HBM-bound: every byte is read once and written once in 16-byte accesses.
// Under FP8 attention each of them also writes the E4M3 codes of every view K row it writes
// (8 bytes per 16-byte granule), and of every view V row under FP8 P V, so the attention's
// operands are ready without another pass.
#include "fk_internal.h"

namespace fk {
namespace {

__device__ __forceinline__ uint4 ld_stream(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
  return v;
}

// plain (coherent) load: the current kernel reads view rows it may itself have written
// in an earlier launch, never in the same launch
__device__ __forceinline__ uint4 ld_plain(const void* p) {
  return *reinterpret_cast<const uint4*>(p);
}

__device__ __forceinline__ void st_v4(void* p, uint4 v) {
  asm volatile("st.global.v4.u32 [%0], {%1,%2,%3,%4};" :: "l"(p), "r"(v.x), "r"(v.y), "r"(v.z),
               "r"(v.w) : "memory");
}

__device__ __forceinline__ int ring_slot(int f, int S, int cap) {
  return f < S ? f : S + (f - S) % cap;
}

// programmatic dependent launch (no-ops for a launch without the programmatic attribute):
// let the next kernel of the stream be scheduled / wait until the previous kernel of the
// stream has completed and its writes are visible
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// Current-chunk update.  A CTA owns TB = 256 / GPR consecutive tokens p of one head h (GPR =
// D/8 16-byte granules per token row) across all C frames of the chunk: thread (p, c) moves
// granule c of rows r*F + p, r < C, of the new chunk (token-major [C*F][H][D], 256 contiguous
// bytes per token and head) into the view front, after copying the previous current chunk's
// granule to its history locations: the page ring (heads that keep history), and the view's
// sink slots and anchor slot (a retired sink frame; the new anchor frame, which every dynamic
// view and, unless they drop it, every static view holds).  Frames go in batches of two with every load of a batch
// issued before its first store.
//
// With a.score set, the CTA also forms the score-contract sums of the retired frames (Eq. 3):
// the GPR lanes of a token hold its GPR channel groups in group order, so the contract's
// per-group fma chains run in each lane and its butterfly p[g] += p[g ^ s], s = GPR/2 .. 1, is a
// lane xor-shuffle; the partner of the first retired frame is the frame before the chunk, read
// from the page ring.  Per (frame, segment) the tokens' int32 halves are summed in shared memory
// and added to the run's int64 sums once per CTA (exact integer adds, order-free).
constexpr int kBatch = 2;
template <int GPR>
__global__ void __launch_bounds__(256, 4) current_kernel(const CurrentArgs a) {
  pdl_trigger();   // the kernel that follows may start its prologue; it waits for this one
  constexpr int TB = 256 / GPR;
  constexpr int D = GPR * 8;
  __shared__ int acc[(kFuseMaxFrames + 1) * TB * 4];   // [frame][segment][N hi, N lo, D hi, D lo]
  const int h = blockIdx.y;
  const int p0 = blockIdx.x * TB;
  const int p = p0 + threadIdx.x / GPR;
  const int c = threadIdx.x % GPR;
  const bool valid = p < a.F;
  const int C = a.rows / a.F;
  const int nh_new = a.nh_old + C;
  const int lo_new = a.W > 0 ? max(a.S, nh_new - a.W) : a.S;
  const int tgt = a.score ? (int)a.score_target[h] : -1;   // uniform over the CTA
  const bool scoring = tgt >= 0;
  const int j0 = p0 / (scoring ? a.seg_len : 1);
  const int segl = valid && scoring ? p / a.seg_len - j0 : 0;   // local segment of token p
  bool bad = false;
  uint4 prev = make_uint4(0, 0, 0, 0);          // the previous frame's granule (contract partner)
  if (scoring) {
    for (int i = threadIdx.x; i < (C + 1) * TB * 4; i += 256) acc[i] = 0;
    if (valid)
      prev = ld_plain(a.pageK[h] + ((int64_t)ring_slot(a.nh_old - 1, a.S, a.cap_nonsink) * a.F + p) * D + c * 8);
    __syncthreads();
    if (a.score_partner_norm) {
      float n = 0.0f, d = 0.0f;
      fma_word(prev.x, prev.x, n, d);
      fma_word(prev.y, prev.y, n, d);
      fma_word(prev.z, prev.z, n, d);
      fma_word(prev.w, prev.w, n, d);
#pragma unroll
      for (int sft = GPR / 2; sft >= 1; sft >>= 1) n = __fadd_rn(n, __shfl_xor_sync(0xffffffffu, n, sft));
      if (valid && c == 0) {
        bad |= !(n <= 8388608.0f);
        int hi, lo;
        fixed24_split(n, hi, lo);
        atomicAdd(&acc[segl * 4 + 0], hi);
        atomicAdd(&acc[segl * 4 + 1], lo);
      }
    }
  }
  for (int r0 = 0; r0 < C; r0 += kBatch) {
    uint4 ko[kBatch], vo[kBatch], kn[kBatch], vn[kBatch];
    // where frame r's old granule goes (page ring, static view slot); frames replaced within
    // the retire are skipped; static views hold the sinks and (unless they drop it) the anchor
    auto to_page = [&](int r) {
      const int f = a.nh_old + r;
      return a.retire && a.pageK[h] != nullptr && (f < a.S || f >= lo_new);
    };
    auto to_slot = [&](int r) {   // every view holds the sinks; dynamic views the new anchor too
      const int f = a.nh_old + r;
      return a.retire && (f < a.S || (f == nh_new - 1 && (!a.is_static[h] || a.static_anchor)));
    };
#pragma unroll
    for (int i = 0; i < kBatch; ++i) {
      ko[i] = vo[i] = kn[i] = vn[i] = make_uint4(0, 0, 0, 0);
      const int r = r0 + i;
      if (r >= C || !valid) continue;
      const int64_t vof = (int64_t)(r * a.F + p) * D + c * 8;
      const bool keep_old = to_page(r) || to_slot(r);
      if (keep_old || scoring) ko[i] = ld_plain(a.viewK[h] + vof);
      if (keep_old) vo[i] = ld_plain(a.viewV[h] + vof);
      if (a.srcK) {
        const size_t src = ((size_t)(r * a.F + p) * a.heads + h) * D + c * 8;
        kn[i] = ld_stream(a.srcK + src);
        vn[i] = ld_stream(a.srcV + src);
      }
    }
#pragma unroll
    for (int i = 0; i < kBatch; ++i) {
      const int r = r0 + i;
      if (r >= C || !valid) continue;
      const int f = a.nh_old + r;
      if (to_page(r)) {
        const int64_t po = ((int64_t)ring_slot(f, a.S, a.cap_nonsink) * a.F + p) * D + c * 8;
        st_v4(a.pageK[h] + po, ko[i]);
        st_v4(a.pageV[h] + po, vo[i]);
      }
      if (to_slot(r)) {
        const int64_t so = ((int64_t)a.rows + (int64_t)(f < a.S ? f : a.S) * a.F + p) * D + c * 8;
        st_v4(a.viewK[h] + so, ko[i]);
        st_v4(a.viewV[h] + so, vo[i]);
        if (a.viewK8[h]) *reinterpret_cast<uint2*>(a.viewK8[h] + so) = e4m3x8(ko[i], 1.0f);
        if (a.viewV8[h]) *reinterpret_cast<uint2*>(a.viewV8[h] + so) = e4m3x8(vo[i], 1.0f);
      }
      if (a.srcK) {
        const int64_t vof = (int64_t)(r * a.F + p) * D + c * 8;
        st_v4(a.viewK[h] + vof, kn[i]);
        st_v4(a.viewV[h] + vof, vn[i]);
        if (a.viewK8[h]) *reinterpret_cast<uint2*>(a.viewK8[h] + vof) = e4m3x8(kn[i], 1.0f);
        if (a.viewV8[h]) *reinterpret_cast<uint2*>(a.viewV8[h] + vof) = e4m3x8(vn[i], 1.0f);
      }
    }
    if (scoring) {
#pragma unroll
      for (int i = 0; i < kBatch; ++i) {
        if (r0 + i >= C) break;                 // uniform over the CTA
        // channel-group partials (one fma chain per lane, channel order), then the butterfly
        float n = 0.0f, d = 0.0f;
        fma_word(ko[i].x, prev.x, n, d);
        fma_word(ko[i].y, prev.y, n, d);
        fma_word(ko[i].z, prev.z, n, d);
        fma_word(ko[i].w, prev.w, n, d);
#pragma unroll
        for (int sft = GPR / 2; sft >= 1; sft >>= 1) {
          n = __fadd_rn(n, __shfl_xor_sync(0xffffffffu, n, sft));
          d = __fadd_rn(d, __shfl_xor_sync(0xffffffffu, d, sft));
        }
        prev = ko[i];
        if (valid && c < 2) {                   // lane 0: N of this frame, lane 1: D with the last
          const float v = c == 0 ? n : d;
          if (c == 0) bad |= !(n <= 8388608.0f);
          int hi, lo;
          fixed24_split(v, hi, lo);
          int* slot = &acc[((r0 + i + 1) * TB + segl) * 4 + 2 * c];
          atomicAdd(slot, hi);
          atomicAdd(slot + 1, lo);
        }
      }
    }
  }
  if (scoring) {
    if (bad) atomicOr(a.status, kStatusRange);
    __syncthreads();
    const int n_loc = min(TB, (min(p0 + TB, a.F) - 1) / a.seg_len - j0 + 1);   // segments here
    for (int i = threadIdx.x; i < (C + 1) * n_loc * 2; i += 256) {
      const int kk = i / (n_loc * 2), rem = i - kk * n_loc * 2;
      const int sl = rem >> 1, which = rem & 1;
      const int hi = acc[(kk * TB + sl) * 4 + 2 * which], lo = acc[(kk * TB + sl) * 4 + 2 * which + 1];
      if (hi == 0 && lo == 0) continue;
      const long long v = (long long)hi * 16777216ll + (long long)lo;
      atomicAdd(a.sums + (((int64_t)tgt * a.max_run + a.score_k0 + kk) * a.n_seg + j0 + sl) * 2 + which,
                (unsigned long long)v);
    }
  }
}

// token-major [rows][H][D] -> dst[h] + row*D.  Consecutive threads read consecutive
// 16-byte granules of the source; each head's destination rows are contiguous.
__global__ void __launch_bounds__(256) scatter_kernel(const ScatterArgs a) {
  const int gpr = a.head_dim / 8;
  const uint32_t per_row = (uint32_t)(a.heads * gpr);
  const uint32_t total = (uint32_t)a.rows * per_row;   // < 2^31 (checked at configuration)
  for (uint32_t g = blockIdx.x * blockDim.x + threadIdx.x; g < total; g += gridDim.x * blockDim.x) {
    const uint32_t row = g / per_row;
    const int rem = (int)(g - row * per_row);
    const int h = rem / gpr;
    const int c = rem - h * gpr;
    const int64_t dst_off = (int64_t)row * a.head_dim + c * 8;
    if (a.dstK[h]) {
      const uint4 k = ld_stream(a.srcK + (size_t)g * 8);
      st_v4(a.dstK[h] + dst_off, k);
      if (a.dstK8[h]) *reinterpret_cast<uint2*>(a.dstK8[h] + dst_off) = e4m3x8(k, 1.0f);
    }
    if (a.dstV[h]) {
      const uint4 v = ld_stream(a.srcV + (size_t)g * 8);
      st_v4(a.dstV[h] + dst_off, v);
      if (a.dstV8[h]) *reinterpret_cast<uint2*>(a.dstV8[h] + dst_off) = e4m3x8(v, 1.0f);
    }
  }
}

// Source and destination element offsets of unit u of a dynamic head's compaction (its u-th
// kept segment to copy, from the target's kept list); false when u is past the layer's units.
// The segment goes to ring slot (rp0 + u) mod kmax of the view's kept-segment ring, after the
// current chunk, the sinks and the anchor (which the current-chunk and prefill kernels write).
__device__ __forceinline__ bool unit_offsets(const CompactArgs& a, const CompactItem& it, int u,
                                             int64_t& src_off, int64_t& dst_off) {
  const int l = it.layer;
  if (u >= a.n_kept_copy[l]) return false;
  const int sid = a.kept[(int64_t)it.target * a.kmax + a.kp0[l] + u];
  const int frame = sid / a.n_seg;
  const int seg = sid - frame * a.n_seg;
  const int slot = (a.rp0[l] + u) % a.kmax;
  const int64_t dst_row = a.CF + (int64_t)a.S * a.F + a.F + (int64_t)slot * a.seg_len;
  src_off = ((int64_t)ring_slot(frame, a.S, a.cap_nonsink) * a.F + (int64_t)seg * a.seg_len) * a.D;
  dst_off = dst_row * a.D;
  return true;
}

// One CTA copies 16 KB of keys and 16 KB of values of one dynamic head's view: one piece of
// one unit (units_per_cta = 1, a unit spans `splits` pieces), or units_per_cta whole small
// units (token-level segments), each thread resolving the unit of every granule it moves.
__global__ void __launch_bounds__(256) compact_kernel(const CompactArgs a) {
  pdl_trigger();
  pdl_wait();      // kept lists and pages come from the kernels before this one
  const CompactItem it = a.items[blockIdx.y];
  if (!a.active[it.layer]) return;
  const int blk = blockIdx.x / a.splits;
  const int piece = blockIdx.x - blk * a.splits;
  const int G = a.units_per_cta;
  const int64_t n = (int64_t)a.seg_len * a.D / 8;      // 16-byte granules per unit and tensor
  constexpr int kPer = kCompactPiece / 16 / 256;         // granules per thread and tensor
  uint4 k[kPer], v[kPer];
  if (G == 1) {
    int64_t src_off, dst_off;
    if (!unit_offsets(a, it, blk, src_off, dst_off)) return;
    const int64_t g0 = (int64_t)piece * (kCompactPiece / 16);
    const uint4* sK = reinterpret_cast<const uint4*>(it.pagesK + src_off);
    const uint4* sV = reinterpret_cast<const uint4*>(it.pagesV + src_off);
    uint4* dK = reinterpret_cast<uint4*>(it.viewK + dst_off);
    uint4* dV = reinterpret_cast<uint4*>(it.viewV + dst_off);
    uint2* dK8 = it.viewK8 ? reinterpret_cast<uint2*>(it.viewK8 + dst_off) : nullptr;
    uint2* dV8 = it.viewV8 ? reinterpret_cast<uint2*>(it.viewV8 + dst_off) : nullptr;
#pragma unroll
    for (int r = 0; r < kPer; ++r) {
      const int64_t i = g0 + threadIdx.x + r * 256;
      if (i < n) {
        k[r] = ld_stream(sK + i);
        v[r] = ld_stream(sV + i);
      }
    }
#pragma unroll
    for (int r = 0; r < kPer; ++r) {
      const int64_t i = g0 + threadIdx.x + r * 256;
      if (i < n) {
        st_v4(dK + i, k[r]);
        st_v4(dV + i, v[r]);
        if (dK8) dK8[i] = e4m3x8(k[r], 1.0f);
        if (dV8) dV8[i] = e4m3x8(v[r], 1.0f);
      }
    }
    return;
  }
  uint4* dK[kPer];
  uint4* dV[kPer];
  int64_t e8[kPer];                                      // element offset of the E4M3 copy
#pragma unroll
  for (int r = 0; r < kPer; ++r) {
    const int64_t gi = threadIdx.x + r * 256;            // granule of this CTA's G units
    dK[r] = nullptr;
    e8[r] = 0;
    int64_t src_off, dst_off;
    if (gi < G * n && unit_offsets(a, it, blk * G + (int)(gi / n), src_off, dst_off)) {
      const int64_t i = gi - (gi / n) * n;
      k[r] = ld_stream(reinterpret_cast<const uint4*>(it.pagesK + src_off) + i);
      v[r] = ld_stream(reinterpret_cast<const uint4*>(it.pagesV + src_off) + i);
      dK[r] = reinterpret_cast<uint4*>(it.viewK + dst_off) + i;
      dV[r] = reinterpret_cast<uint4*>(it.viewV + dst_off) + i;
      e8[r] = dst_off + i * 8;
    }
  }
#pragma unroll
  for (int r = 0; r < kPer; ++r) {
    if (dK[r]) {
      st_v4(dK[r], k[r]);
      st_v4(dV[r], v[r]);
      if (it.viewK8) *reinterpret_cast<uint2*>(it.viewK8 + e8[r]) = e4m3x8(k[r], 1.0f);
      if (it.viewV8) *reinterpret_cast<uint2*>(it.viewV8 + e8[r]) = e4m3x8(v[r], 1.0f);
    }
  }
}

// Streaming read of `n` 16-byte granules (calibration of the HBM-bound kernels): a grid-stride
// loop with four loads in flight per thread and no other work; the xor of the data decides a
// store that never happens for the bench's data, so the loads cannot be removed.
__device__ unsigned g_read_sink;
__global__ void __launch_bounds__(256) stream_read_kernel(const uint4* __restrict__ src, int64_t n) {
  uint32_t acc = 0;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  for (; i + 3 * stride < n; i += 4 * stride) {
    const uint4 v0 = ld_stream(src + i), v1 = ld_stream(src + i + stride);
    const uint4 v2 = ld_stream(src + i + 2 * stride), v3 = ld_stream(src + i + 3 * stride);
    acc ^= v0.x ^ v1.y ^ v2.z ^ v3.w;
  }
  for (; i < n; i += stride) acc ^= ld_stream(src + i).x;
  if (acc == 0x5EEDF00Du) atomicAdd(&g_read_sink, 1u);
}

unsigned grid_for(int64_t granules) {
  int64_t blocks = (granules + 255) / 256;
  if (blocks > 152 * 16) blocks = 152 * 16;
  return (unsigned)(blocks < 1 ? 1 : blocks);
}

}  // namespace

void launch_current(const CurrentArgs& a, cudaStream_t s) {
  if (a.rows == 0 || a.heads == 0) return;
  const int gpr = a.head_dim / 8, tb = 256 / gpr;
  const dim3 grid((unsigned)((a.F + tb - 1) / tb), (unsigned)a.heads);
  if (gpr == 16) current_kernel<16><<<grid, 256, 0, s>>>(a);
  else current_kernel<8><<<grid, 256, 0, s>>>(a);
}

void launch_scatter(const ScatterArgs& a, cudaStream_t s) {
  const int64_t total = (int64_t)a.rows * a.heads * (a.head_dim / 8);
  if (total == 0) return;
  scatter_kernel<<<grid_for(total), 256, 0, s>>>(a);
}

void launch_compact(const CompactArgs& a, cudaStream_t s) {
  if (a.n_items == 0 || a.max_units == 0) return;
  // programmatic launch: the grid is scheduled while the selection kernel runs
  cudaLaunchConfig_t cfg{};
  const int blocks = (a.max_units + a.units_per_cta - 1) / a.units_per_cta;
  cfg.gridDim = dim3((unsigned)(blocks * a.splits), (unsigned)a.n_items);
  cfg.blockDim = dim3(256);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaLaunchKernelEx(&cfg, compact_kernel, a);
}

cudaError_t launch_stream_read(const void* src, int64_t bytes, cudaStream_t s) {
  if (bytes <= 0) return cudaSuccess;
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  stream_read_kernel<<<sms * 8, 256, 0, s>>>(static_cast<const uint4*>(src), bytes / 16);
  return cudaGetLastError();
}

}  // namespace fk
