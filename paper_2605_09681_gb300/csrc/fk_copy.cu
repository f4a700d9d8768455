// Data-movement kernels of the Forcing-KV cache: the current chunk's scatter from the
// caller's token-major [tokens][H][D] layout into per-head views, frame copies into the
// history pages (append), and the select-and-compact gather of kept segments into the
// packed per-head views of dynamic heads (Sec. 4.3, Eq. 4: [sink, kept segments, anchor]).
// All three are HBM-bound: every byte is read once and written once with 16-byte accesses.
#include "fk_internal.h"

namespace fk {
namespace {

__device__ __forceinline__ uint4 ld_stream(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
  return v;
}

__device__ __forceinline__ void st_v4(void* p, uint4 v) {
  asm volatile("st.global.v4.u32 [%0], {%1,%2,%3,%4};" :: "l"(p), "r"(v.x), "r"(v.y), "r"(v.z),
               "r"(v.w) : "memory");
}

// token-major [rows][H][D] -> dst[h] + row*D.  Consecutive threads read consecutive
// 16-byte granules of the source; each head's destination rows are contiguous.
__global__ void __launch_bounds__(256) scatter_kernel(const ScatterArgs a) {
  const int gpr = a.head_dim / 8;                       // granules per head row
  const int64_t per_row = (int64_t)a.heads * gpr;
  const int64_t total = (int64_t)a.rows * per_row;
  for (int64_t g = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; g < total;
       g += (int64_t)gridDim.x * blockDim.x) {
    const int64_t row = g / per_row;
    const int rem = (int)(g - row * per_row);
    const int h = rem / gpr;
    const int c = rem - h * gpr;
    const int64_t dst_off = row * a.head_dim + c * 8;
    if (a.dstK[h]) st_v4(a.dstK[h] + dst_off, ld_stream(a.srcK + g * 8));
    if (a.dstV[h]) st_v4(a.dstV[h] + dst_off, ld_stream(a.srcV + g * 8));
  }
}

// a list of contiguous copies; blockIdx.y selects the job
__global__ void __launch_bounds__(256) copy_jobs_kernel(const CopyJobs j) {
  const CopyJob& job = j.job[blockIdx.y];
  const int64_t n = job.bytes / 16;
  const uint4* src = static_cast<const uint4*>(job.src);
  uint4* dst = static_cast<uint4*>(job.dst);
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  for (; i + 3 * stride < n; i += 4 * stride) {
    uint4 v0 = ld_stream(src + i), v1 = ld_stream(src + i + stride);
    uint4 v2 = ld_stream(src + i + 2 * stride), v3 = ld_stream(src + i + 3 * stride);
    st_v4(dst + i, v0); st_v4(dst + i + stride, v1);
    st_v4(dst + i + 2 * stride, v2); st_v4(dst + i + 3 * stride, v3);
  }
  for (; i < n; i += stride) st_v4(dst + i, ld_stream(src + i));
}

__device__ __forceinline__ int ring_slot(int f, int S, int cap) {
  return f < S ? f : S + (f - S) % cap;
}

// One CTA copies one unit (F/n tokens of keys and values) of one dynamic head's view.
// Units in view order: sink frames (n units each), kept segments (ascending t*n+j),
// anchor frame (n units).  Unit u lands at view row CF + u*seg_len.
__global__ void __launch_bounds__(256) compact_kernel(const CompactArgs a) {
  const CompactItem it = a.items[blockIdx.y];
  const int l = it.layer;
  if (!a.active[l]) return;
  const int u = blockIdx.x;
  const int n_sink_units = a.n_sink_present[l] * a.n_seg;
  const int n_keep = a.n_keep[l];
  const int units = n_sink_units + n_keep + (a.anchor[l] >= 0 ? a.n_seg : 0);
  if (u >= units) return;
  int frame, seg;
  if (u < n_sink_units) {
    frame = u / a.n_seg;
    seg = u - frame * a.n_seg;
  } else if (u < n_sink_units + n_keep) {
    const int sid = a.kept[(int64_t)it.target * a.kmax + (u - n_sink_units)];
    frame = sid / a.n_seg;
    seg = sid - frame * a.n_seg;
  } else {
    frame = a.anchor[l];
    seg = u - n_sink_units - n_keep;
  }
  const int slot = ring_slot(frame, a.S, a.cap_nonsink);
  const int64_t src_off = ((int64_t)slot * a.F + (int64_t)seg * a.seg_len) * a.D;
  const int64_t dst_off = ((int64_t)a.CF + (int64_t)u * a.seg_len) * a.D;
  const int64_t n = (int64_t)a.seg_len * a.D / 8;      // 16-byte granules per tensor
  const uint4* sK = reinterpret_cast<const uint4*>(it.pagesK + src_off);
  const uint4* sV = reinterpret_cast<const uint4*>(it.pagesV + src_off);
  uint4* dK = reinterpret_cast<uint4*>(it.viewK + dst_off);
  uint4* dV = reinterpret_cast<uint4*>(it.viewV + dst_off);
  int64_t i = threadIdx.x;
  for (; i + 256 < n; i += 512) {
    uint4 k0 = ld_stream(sK + i), k1 = ld_stream(sK + i + 256);
    uint4 v0 = ld_stream(sV + i), v1 = ld_stream(sV + i + 256);
    st_v4(dK + i, k0); st_v4(dK + i + 256, k1);
    st_v4(dV + i, v0); st_v4(dV + i + 256, v1);
  }
  for (; i < n; i += 256) {
    st_v4(dK + i, ld_stream(sK + i));
    st_v4(dV + i, ld_stream(sV + i));
  }
}

}  // namespace

void launch_scatter(const ScatterArgs& a, cudaStream_t s) {
  const int64_t total = (int64_t)a.rows * a.heads * (a.head_dim / 8);
  if (total == 0) return;
  int64_t blocks = (total + 255) / 256;
  if (blocks > 152 * 16) blocks = 152 * 16;
  scatter_kernel<<<(unsigned)blocks, 256, 0, s>>>(a);
}

void launch_copy_jobs(const CopyJobs& j, cudaStream_t s) {
  if (j.n == 0) return;
  int64_t maxb = 0;
  for (int i = 0; i < j.n; ++i) maxb = j.job[i].bytes > maxb ? j.job[i].bytes : maxb;
  int64_t bx = (maxb / 16 + 1023) / 1024;
  if (bx < 1) bx = 1;
  if (bx > 64) bx = 64;
  copy_jobs_kernel<<<dim3((unsigned)bx, (unsigned)j.n), 256, 0, s>>>(j);
}

void launch_compact(const CompactArgs& a, cudaStream_t s) {
  if (a.n_items == 0 || a.max_units == 0) return;
  compact_kernel<<<dim3((unsigned)a.max_units, (unsigned)a.n_items), 256, 0, s>>>(a);
}

}  // namespace fk
