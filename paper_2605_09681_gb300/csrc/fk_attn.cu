// Chunk attention over the per-head packed views (Sec. 4.2 Eq. 2, Sec. 4.3 Eq. 4):
// O = softmax(Q K^T / sqrt(D)) V per head, with a different key count per head.
//
// One CTA computes 128 query rows of one head against all of the head's keys, in
// tiles of 128 keys, on the 5th-generation tensor cores:
//   warp 4 (one lane)  TMA: Q once (3D map over [Nq][H][D]), K and V tiles (2D maps over
//                      the view arenas) into a two-stage ring, 128-byte swizzle;
//   warp 5 (one lane)  tcgen05.mma: S = Q K^T into one of two TMEM buffers, then
//                      O += P V into a TMEM accumulator; completion via tcgen05.commit;
//   warps 0-3          softmax: thread r owns query row r = TMEM lane r; reads S with
//                      tcgen05.ld, online softmax in the log2 domain with a lazily
//                      rescaled running max, writes P (bf16) to shared memory for the
//                      second MMA, and finally normalises O and stores it.
// Every mbarrier wait is bounded (%globaltimer); on expiry the CTA records
// FK_ERR_TIMEOUT in the status word, drains its own TMA loads and MMAs and frees TMEM.
#include "fk_internal.h"

namespace fk {
namespace {

constexpr uint64_t kWaitLimitNs = 2000000000ull;   // 2 s per wait
constexpr float kRescaleThreshold = 8.0f;          // log2 units: rescale O when max grows > 2^8

struct AttnBarriers {
  uint64_t q_full;
  uint64_t k_full[2], k_empty[2];
  uint64_t v_full[2], v_empty[2];
  uint64_t s_full[2], s_free[2];
  uint64_t p_full, pv_done, fin;
  uint32_t tmem_base;
  volatile int abort;
};

template <int D>
struct Layout {
  static constexpr int kQ = kAttnBM * D * 2;
  static constexpr int kKV = kAttnBN * D * 2;
  static constexpr int kP = kAttnBM * kAttnBN * 2;
  static constexpr int kOffQ = 0;
  static constexpr int kOffK = kOffQ + kQ;
  static constexpr int kOffV = kOffK + 2 * kKV;
  static constexpr int kOffP = kOffV + 2 * kKV;
  static constexpr int kOffBar = kOffP + kP;
  static constexpr int kUsed = kOffBar + 256;
  // at least ~116 KB so that one CTA occupies an SM (its 512 TMEM columns are then free)
  static constexpr int kSmem = (kUsed + 1024) > 118 * 1024 ? (kUsed + 1024) : 118 * 1024;
};

__device__ __forceinline__ uint32_t su32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t now_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void mbar_init(uint64_t* b, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" :: "r"(su32(b)), "r"(count));
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* b, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" :: "r"(su32(b)),
               "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* b) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" :: "r"(su32(b)) : "memory");
}
__device__ __forceinline__ bool mbar_test(uint64_t* b, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok) : "r"(su32(b)), "r"(parity) : "memory");
  return ok != 0;
}

// Bounded wait for the phase of parity `parity`.  Returns false when the CTA is
// aborting or the limit expired (which starts the abort).
__device__ __noinline__ bool wait_phase(uint64_t* b, uint32_t parity, AttnBarriers* bar,
                                        int* status, bool honour_abort = true) {
  if (mbar_test(b, parity)) return true;
  const uint64_t t0 = now_ns();
  while (true) {
    if (mbar_test(b, parity)) return true;
    if (honour_abort && bar->abort) return false;
    if (now_ns() - t0 > kWaitLimitNs) {
      bar->abort = 1;
      atomicOr(status, kStatusTimeout);
      return false;
    }
  }
}

// Warp-uniform bounded wait: every lane polls, and the warp proceeds only if all did.
__device__ __forceinline__ bool warp_wait(uint64_t* b, uint32_t parity, AttnBarriers* bar,
                                          int* status) {
  const bool ok = wait_phase(b, parity, bar, status);
  return __all_sync(0xffffffffu, ok);
}

__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, uint64_t* b,
                                            int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4}], [%2];"
      :: "r"(su32(dst)), "l"(map), "r"(su32(b)), "r"(x), "r"(y) : "memory");
}
__device__ __forceinline__ void tma_load_3d(void* dst, const CUtensorMap* map, uint64_t* b,
                                            int x, int y, int z) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4, %5}], [%2];"
      :: "r"(su32(dst)), "l"(map), "r"(su32(b)), "r"(x), "r"(y), "r"(z) : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// Shared-memory matrix descriptor (tcgen05): start, leading/stride byte offsets (16-byte
// units), descriptor version 1, 128-byte swizzle.
__device__ __forceinline__ uint64_t sdesc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  return (uint64_t)((saddr >> 4) & 0x3FFFu) | ((uint64_t)((lbo >> 4) & 0x3FFFu) << 16) |
         ((uint64_t)((sbo >> 4) & 0x3FFFu) << 32) | (1ull << 46) | (2ull << 61);
}

// Instruction descriptor, kind::f16: f32 accumulate, bf16 A and B, A K-major,
// B K-major (b_mn = 0) or MN-major (b_mn = 1), N >> 3 at bit 17, M >> 4 at bit 24.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N, int b_mn) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)b_mn << 16) |
         ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

__device__ __forceinline__ void umma(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                     uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n"
      :: "r"(d_tmem), "l"(a), "l"(b), "r"(idesc), "r"(accumulate) : "memory");
}
__device__ __forceinline__ void umma_commit(uint64_t* b) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];"
      :: "r"(su32(b)) : "memory");
}

#define FK_TMEM_LD32(taddr, v)                                                              \
  asm volatile(                                                                             \
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,"  \
      "%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];" \
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),  \
        "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]),           \
        "=r"(v[13]), "=r"(v[14]), "=r"(v[15]), "=r"(v[16]), "=r"(v[17]), "=r"(v[18]),        \
        "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]),        \
        "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]),        \
        "=r"(v[31])                                                                         \
      : "r"(taddr))

#define FK_TMEM_ST32(taddr, v)                                                              \
  asm volatile(                                                                             \
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,"   \
      "%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" \
      :: "r"(taddr), "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]),      \
        "r"(v[6]), "r"(v[7]), "r"(v[8]), "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]),      \
        "r"(v[13]), "r"(v[14]), "r"(v[15]), "r"(v[16]), "r"(v[17]), "r"(v[18]), "r"(v[19]),  \
        "r"(v[20]), "r"(v[21]), "r"(v[22]), "r"(v[23]), "r"(v[24]), "r"(v[25]), "r"(v[26]),  \
        "r"(v[27]), "r"(v[28]), "r"(v[29]), "r"(v[30]), "r"(v[31]) : "memory")

__device__ __forceinline__ void tmem_wait_ld() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_wait_st() {
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  const __nv_bfloat162 p = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&p);
}

template <int D>
__global__ void __launch_bounds__(192, 1)
attn_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
            const __grid_constant__ CUtensorMap tmV, const AttnArgs a) {
  using Lay = Layout<D>;
  constexpr int kHalves = D / 64;                 // 64-column (128-byte) swizzle atoms
  constexpr uint32_t kTmemCols = 512;
  constexpr uint32_t kColO = 2 * kAttnBN;         // S0 = cols 0..127, S1 = 128..255, O = 256..
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* sQ = smem + Lay::kOffQ;
  uint8_t* sK = smem + Lay::kOffK;
  uint8_t* sV = smem + Lay::kOffV;
  uint8_t* sP = smem + Lay::kOffP;
  AttnBarriers* bar = reinterpret_cast<AttnBarriers*>(smem + Lay::kOffBar);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int hi = blockIdx.x / a.n_qtiles;
  const int q0 = (blockIdx.x - hi * a.n_qtiles) * kAttnBM;
  const int head = a.head_of[hi];
  const int nk = a.n_keys[head];
  const int row0 = a.row_base[head];
  const int nt = (nk + kAttnBN - 1) / kAttnBN;

  if (threadIdx.x == 0) {
    mbar_init(&bar->q_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bar->k_full[i], 1);
      mbar_init(&bar->k_empty[i], 1);
      mbar_init(&bar->v_full[i], 1);
      mbar_init(&bar->v_empty[i], 1);
      mbar_init(&bar->s_full[i], 1);
      mbar_init(&bar->s_free[i], 4);
    }
    mbar_init(&bar->p_full, 4);
    mbar_init(&bar->pv_done, 1);
    mbar_init(&bar->fin, 1);
    bar->abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 5) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;"
                 :: "r"(su32(&bar->tmem_base)), "r"(kTmemCols) : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bar->tmem_base;

  if (warp == 4) {
    // ------------------------------------------------------------------ TMA producer
    if (lane == 0) {
      int lastK[2] = {-1, -1}, lastV[2] = {-1, -1};
      bool ok = true;
      mbar_expect_tx(&bar->q_full, Lay::kQ);
      for (int h = 0; h < kHalves; ++h)
        tma_load_3d(sQ + h * 16384, &tmQ, &bar->q_full, h * 64, head, q0);
      for (int j = 0; j < nt && ok; ++j) {
        const int st = j & 1, u = j >> 1;
        if (j >= 2 && !wait_phase(&bar->k_empty[st], (u - 1) & 1, bar, a.status)) { ok = false; break; }
        mbar_expect_tx(&bar->k_full[st], Lay::kKV);
        for (int h = 0; h < kHalves; ++h)
          tma_load_2d(sK + st * Lay::kKV + h * 16384, &tmK, &bar->k_full[st], h * 64,
                      row0 + j * kAttnBN);
        lastK[st] = u;
        if (j >= 2 && !wait_phase(&bar->v_empty[st], (u - 1) & 1, bar, a.status)) { ok = false; break; }
        mbar_expect_tx(&bar->v_full[st], Lay::kKV);
        for (int h = 0; h < kHalves; ++h)
          tma_load_2d(sV + st * Lay::kKV + h * 16384, &tmV, &bar->v_full[st], h * 64,
                      row0 + j * kAttnBN);
        lastV[st] = u;
      }
      if (!ok) {   // drain every load this thread issued before the CTA exits
        wait_phase(&bar->q_full, 0, bar, a.status, false);
        for (int st = 0; st < 2; ++st) {
          if (lastK[st] >= 0) wait_phase(&bar->k_full[st], lastK[st] & 1, bar, a.status, false);
          if (lastV[st] >= 0) wait_phase(&bar->v_full[st], lastV[st] & 1, bar, a.status, false);
        }
      }
    }
    __syncwarp();
  } else if (warp == 5) {
    // ------------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t kIdQK = idesc_bf16(kAttnBM, kAttnBN, 0);
      constexpr uint32_t kIdPV = idesc_bf16(kAttnBM, D, 1);
      const uint32_t aQ = su32(sQ), aK = su32(sK), aV = su32(sV), aP = su32(sP);
      auto pv = [&](int i) -> bool {
        const int st = i & 1;
        if (!wait_phase(&bar->p_full, i & 1, bar, a.status)) return false;
        if (!wait_phase(&bar->v_full[st], (i >> 1) & 1, bar, a.status)) return false;
        tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < kAttnBN / 16; ++kk) {
          const uint64_t da = sdesc(aP + (kk >> 2) * 16384 + (kk & 3) * 32, 16, 1024);
          const uint64_t db = sdesc(aV + st * Lay::kKV + kk * 2048, 16384, 1024);
          umma(tmem + kColO, da, db, kIdPV, (i > 0 || kk > 0) ? 1u : 0u);
        }
        umma_commit(&bar->v_empty[st]);
        umma_commit(&bar->pv_done);
        return true;
      };
      bool ok = wait_phase(&bar->q_full, 0, bar, a.status);
      for (int j = 0; j < nt && ok; ++j) {
        const int st = j & 1, u = j >> 1;
        if (!wait_phase(&bar->k_full[st], u & 1, bar, a.status)) { ok = false; break; }
        if (j >= 2 && !wait_phase(&bar->s_free[j & 1], (u - 1) & 1, bar, a.status)) { ok = false; break; }
        tc_fence_after();
        const uint32_t tS = tmem + (uint32_t)((j & 1) * kAttnBN);
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint64_t da = sdesc(aQ + (kk >> 2) * 16384 + (kk & 3) * 32, 16, 1024);
          const uint64_t db = sdesc(aK + st * Lay::kKV + (kk >> 2) * 16384 + (kk & 3) * 32, 16, 1024);
          umma(tS, da, db, kIdQK, kk > 0 ? 1u : 0u);
        }
        umma_commit(&bar->s_full[j & 1]);
        umma_commit(&bar->k_empty[st]);
        if (j >= 1 && !pv(j - 1)) { ok = false; break; }
      }
      if (ok) pv(nt - 1);
      umma_commit(&bar->fin);                       // completes once every MMA above is done
      wait_phase(&bar->fin, 0, bar, a.status, false);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------------ softmax warps 0-3
    const int row = warp * 32 + lane;
    const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
    float m = -INFINITY, l = 0.0f;
    bool ok = true;
    for (int j = 0; j < nt; ++j) {
      if (!warp_wait(&bar->s_full[j & 1], (j >> 1) & 1, bar, a.status)) { ok = false; break; }
      tc_fence_after();
      float s[kAttnBN];
      {
        uint32_t* sv = reinterpret_cast<uint32_t*>(s);
        const uint32_t tS = tmem + lane_base + (uint32_t)((j & 1) * kAttnBN);
        FK_TMEM_LD32(tS + 0, (sv + 0));
        FK_TMEM_LD32(tS + 32, (sv + 32));
        FK_TMEM_LD32(tS + 64, (sv + 64));
        FK_TMEM_LD32(tS + 96, (sv + 96));
        tmem_wait_ld();
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bar->s_free[j & 1]);

      const int valid = nk - j * kAttnBN;
      if (valid < kAttnBN) {
#pragma unroll
        for (int c = 0; c < kAttnBN; ++c)
          if (c >= valid) s[c] = -INFINITY;
      }
      float mx = s[0];
#pragma unroll
      for (int c = 1; c < kAttnBN; ++c) mx = fmaxf(mx, s[c]);
      const float m_new = fmaxf(m, mx * a.scale_log2);
      bool pv_waited = false;
      const bool need = m_new > m + kRescaleThreshold;
      if (__any_sync(0xffffffffu, need)) {
        const float alpha = fast_exp2(m - m_new);    // 0 when m = -inf
        if (j > 0) {
          if (!warp_wait(&bar->pv_done, (j - 1) & 1, bar, a.status)) { ok = false; break; }
          pv_waited = true;
          tc_fence_after();
#pragma unroll
          for (int c = 0; c < D / 32; ++c) {
            uint32_t o[32];
            const uint32_t tO = tmem + lane_base + kColO + c * 32;
            FK_TMEM_LD32(tO, o);
            tmem_wait_ld();
#pragma unroll
            for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
            FK_TMEM_ST32(tO, o);
          }
          tmem_wait_st();
        }
        l *= alpha;
        m = m_new;
      }
      float rs = 0.0f;
#pragma unroll
      for (int c = 0; c < kAttnBN; ++c) {
        s[c] = fast_exp2(fmaf(s[c], a.scale_log2, -m));
        rs += s[c];
      }
      l += rs;
      if (j > 0 && !pv_waited) {
        if (!warp_wait(&bar->pv_done, (j - 1) & 1, bar, a.status)) { ok = false; break; }
      }
      // P row -> shared memory, K-major with the 128-byte swizzle (chunk ^= row % 8)
      uint8_t* prow = sP + row * 128;
#pragma unroll
      for (int cc = 0; cc < kAttnBN / 8; ++cc) {
        uint4 v;
        v.x = pack_bf16(s[cc * 8 + 0], s[cc * 8 + 1]);
        v.y = pack_bf16(s[cc * 8 + 2], s[cc * 8 + 3]);
        v.z = pack_bf16(s[cc * 8 + 4], s[cc * 8 + 5]);
        v.w = pack_bf16(s[cc * 8 + 6], s[cc * 8 + 7]);
        const int atom = cc >> 3, ch = (cc & 7) ^ (row & 7);
        *reinterpret_cast<uint4*>(prow + atom * 16384 + ch * 16) = v;
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bar->p_full);
    }
    // ---------------------------------------------------------------- epilogue
    if (ok && warp_wait(&bar->pv_done, (nt - 1) & 1, bar, a.status)) {
      tc_fence_after();
      const float inv = 1.0f / l;
      const int q = q0 + row;
      bf16* orow = a.O + ((int64_t)q * a.H + head) * D;
#pragma unroll
      for (int c = 0; c < D / 32; ++c) {
        uint32_t o[32];
        FK_TMEM_LD32(tmem + lane_base + kColO + c * 32, o);
        tmem_wait_ld();
        if (q < a.Nq) {
#pragma unroll
          for (int e = 0; e < 32; e += 8) {
            uint4 v;
            v.x = pack_bf16(__uint_as_float(o[e + 0]) * inv, __uint_as_float(o[e + 1]) * inv);
            v.y = pack_bf16(__uint_as_float(o[e + 2]) * inv, __uint_as_float(o[e + 3]) * inv);
            v.z = pack_bf16(__uint_as_float(o[e + 4]) * inv, __uint_as_float(o[e + 5]) * inv);
            v.w = pack_bf16(__uint_as_float(o[e + 6]) * inv, __uint_as_float(o[e + 7]) * inv);
            *reinterpret_cast<uint4*>(orow + c * 32 + e) = v;
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 5) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" :: "r"(tmem),
                 "r"(kTmemCols) : "memory");
  }
}

}  // namespace

cudaError_t attention_prepare(int head_dim) {
  if (head_dim == 128)
    return cudaFuncSetAttribute(attn_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                Layout<128>::kSmem);
  return cudaFuncSetAttribute(attn_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              Layout<64>::kSmem);
}

void launch_attention(int head_dim, const CUtensorMap& tmQ, const CUtensorMap& tmK,
                      const CUtensorMap& tmV, const AttnArgs& a, cudaStream_t s) {
  const unsigned grid = (unsigned)(a.n_qtiles * a.H);
  if (head_dim == 128)
    attn_kernel<128><<<grid, 192, Layout<128>::kSmem, s>>>(tmQ, tmK, tmV, a);
  else
    attn_kernel<64><<<grid, 192, Layout<64>::kSmem, s>>>(tmQ, tmK, tmV, a);
}

}  // namespace fk
