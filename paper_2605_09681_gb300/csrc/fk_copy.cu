// Data-movement kernels of the Forcing-KV cache: the current-chunk update (the previous
// current chunk joins the history pages and the new chunk is scattered from the caller's
// token-major [tokens][H][D] layout into the per-head views, in one pass), the prefill
// scatter of history frames, and the select-and-compact gather of kept segments into the
// packed per-head views of dynamic heads (Sec. 4.3, Eq. 4: sink, kept segments and the
// anchor frame; attention does not depend on the order of the keys, so a view holds them as
// [sinks | anchor | kept-segment ring] and incremental compaction only appends).
// All of them are HBM-bound: every byte is read once and written once in 16-byte accesses.
// Under FP8_QK attention each of them also writes the E4M3 codes of every view K row it writes
// (8 bytes per 16-byte granule), so the attention's key operand is ready without another pass.
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

// One thread per 16-byte granule of the current chunk, indexed in the caller's token-major
// order (row, head, granule) so that the reads of the new chunk are fully coalesced.
__global__ void __launch_bounds__(256) current_kernel(const CurrentArgs a) {
  pdl_trigger();   // the scoring kernel that follows may start its prologue; it waits for us
  const int gpr = a.head_dim / 8;
  const uint32_t per_row = (uint32_t)(a.heads * gpr);
  const uint32_t total = (uint32_t)a.rows * per_row;   // < 2^31 (checked at configuration)
  const int nh_new = a.nh_old + a.rows / a.F;
  const int lo_new = a.W > 0 ? max(a.S, nh_new - a.W) : a.S;
  for (uint32_t g = blockIdx.x * blockDim.x + threadIdx.x; g < total; g += gridDim.x * blockDim.x) {
    const int row = (int)(g / per_row);
    const int rem = (int)(g - row * per_row);
    const int h = rem / gpr;
    const int c = rem - h * gpr;
    const int64_t vo = (int64_t)row * a.head_dim + c * 8;
    bool to_page = false, to_slot = false;
    int64_t po = 0, so = 0;
    if (a.retire) {
      const int f = a.nh_old + row / a.F;
      const int p = row - (row / a.F) * a.F;
      const bool sink = f < a.S;
      // frames replaced within the retire are skipped; static views hold the sinks and
      // (unless they drop it) the new anchor frame
      to_page = a.pageK[h] != nullptr && (sink || f >= lo_new);
      to_slot = a.is_static[h] && (sink || (a.static_anchor && f == nh_new - 1));
      po = ((int64_t)ring_slot(f, a.S, a.cap_nonsink) * a.F + p) * a.head_dim + c * 8;
      so = ((int64_t)a.rows + (int64_t)(sink ? f : a.S) * a.F + p) * a.head_dim + c * 8;
    }
    // every load first (old granule, new granule), then the stores
    uint4 ko = make_uint4(0, 0, 0, 0), vo4 = ko, kn = ko, vn = ko;
    if (to_page || to_slot) {
      ko = ld_plain(a.viewK[h] + vo);
      vo4 = ld_plain(a.viewV[h] + vo);
    }
    if (a.srcK) {
      kn = ld_stream(a.srcK + (size_t)g * 8);
      vn = ld_stream(a.srcV + (size_t)g * 8);
    }
    if (to_page) {
      st_v4(a.pageK[h] + po, ko);
      st_v4(a.pageV[h] + po, vo4);
    }
    if (to_slot) {
      st_v4(a.viewK[h] + so, ko);
      st_v4(a.viewV[h] + so, vo4);
      if (a.viewK8[h]) *reinterpret_cast<uint2*>(a.viewK8[h] + so) = e4m3x8(ko, 1.0f);
    }
    if (a.srcK) {
      st_v4(a.viewK[h] + vo, kn);
      st_v4(a.viewV[h] + vo, vn);
      if (a.viewK8[h]) *reinterpret_cast<uint2*>(a.viewK8[h] + vo) = e4m3x8(kn, 1.0f);
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
    if (a.dstV[h]) st_v4(a.dstV[h] + dst_off, ld_stream(a.srcV + (size_t)g * 8));
  }
}

// Source and destination element offsets of unit u of a dynamic head's compaction; false
// when u is past the layer's units.  Units in order: the sink frames to copy (n units each),
// the anchor frame (n units), the kept segments to copy (one unit each, from the target's kept
// list).  View rows after the current chunk: sink frame f at S-slot f, the anchor after the
// sinks, kept segment i in ring slot (rp0 + i) mod kmax after the anchor.
__device__ __forceinline__ bool unit_offsets(const CompactArgs& a, const CompactItem& it, int u,
                                             int64_t& src_off, int64_t& dst_off) {
  const int l = it.layer;
  const int n_sink_units = a.n_sink_copy[l] * a.n_seg;
  const int n_anchor_units = a.anchor[l] >= 0 ? a.n_seg : 0;
  if (u >= n_sink_units + n_anchor_units + a.n_kept_copy[l]) return false;
  int frame, seg;
  int64_t dst_row = a.CF;
  if (u < n_sink_units) {
    frame = a.sink_first[l] + u / a.n_seg;
    seg = u - (u / a.n_seg) * a.n_seg;
    dst_row += (int64_t)frame * a.F + (int64_t)seg * a.seg_len;
  } else if (u < n_sink_units + n_anchor_units) {
    frame = a.anchor[l];
    seg = u - n_sink_units;
    dst_row += (int64_t)a.S * a.F + (int64_t)seg * a.seg_len;
  } else {
    const int i = u - n_sink_units - n_anchor_units;
    const int sid = a.kept[(int64_t)it.target * a.kmax + a.kp0[l] + i];
    frame = sid / a.n_seg;
    seg = sid - frame * a.n_seg;
    const int slot = (a.rp0[l] + i) % a.kmax;
    dst_row += (int64_t)a.S * a.F + a.F + (int64_t)slot * a.seg_len;
  }
  const int slot = ring_slot(frame, a.S, a.cap_nonsink);
  src_off = ((int64_t)slot * a.F + (int64_t)seg * a.seg_len) * a.D;
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
    }
  }
}

unsigned grid_for(int64_t granules) {
  int64_t blocks = (granules + 255) / 256;
  if (blocks > 152 * 16) blocks = 152 * 16;
  return (unsigned)(blocks < 1 ? 1 : blocks);
}

}  // namespace

void launch_current(const CurrentArgs& a, cudaStream_t s) {
  const int64_t total = (int64_t)a.rows * a.heads * (a.head_dim / 8);
  if (total == 0) return;
  current_kernel<<<grid_for(total), 256, 0, s>>>(a);
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

}  // namespace fk
