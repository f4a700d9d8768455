// Chunk attention over the per-head packed views (Sec. 4.2 Eq. 2, Sec. 4.3 Eq. 4):
// O = softmax(Q K^T / sqrt(D)) V per head, with a different key count per head.
//
// One CTA computes two 128-row query tiles of one head against all of the head's keys,
// in tiles of 128 keys, on the 5th-generation tensor cores:
//   warp 8 (one lane)  TMA: both Q tiles once (3D map over [Nq][H][D]), K and V tiles (2D
//                      maps over the view arenas) into two-stage rings, 128-byte swizzle;
//                      key tile 0 on its own barrier, then V_j together with K_{j+1} on one
//                      barrier per stage pair (one wait and one release per key tile);
//   warp 9 (one lane)  tcgen05.mma, per key tile j: P_0 V_j, S_0(j+1), P_1 V_j, S_1(j+1)
//                      (S_t = Q_t K^T into TMEM, O_t += P_t V with P_t read from TMEM);
//                      completion via tcgen05.commit; the barriers of the next group are
//                      tested without blocking while the tensor pipe still runs this one;
//   warps 0-3 / 4-7    softmax of query tile 0 / 1 (ping-pong: one warpgroup's softmax
//                      overlaps the other tile's MMAs): thread r owns row r = TMEM lane r,
//                      reads S with tcgen05.ld, online softmax in the log2 domain with a
//                      lazily rescaled running max, writes P as bf16 pairs over S's first
//                      64 columns with tcgen05.st, and finally normalises O and stores it.
//                      After the first key tile a 64-key half computes P with the running
//                      max at once; its sum (at most 2^8) or the packed maximum of its P
//                      shows that no numerator exceeds the rescale bound, else the half is
//                      redone with a max pass.
// TMEM columns: S0 0-127, S1 128-255, O0 256.., O1 256+D.. (512 allocated).
// FP8_QK variant (D = 128): the K tiles hold E4M3 codes (one 128-byte swizzle atom per row,
// from the view arena's E4M3 copy); the bf16 Q tiles are loaded as usual and each softmax
// thread quantizes its own row into an E4M3 tile (row exponent e_row, codes of the row times
// 2^-e_row, written in the 128-byte swizzle pattern) before the first MMA; S = Q K^T runs as
// tcgen05.mma kind::f8f6f4 (K = 32 per instruction) and the thread scales its row's logits by
// 2^e_row along with 1/sqrt(D); P V is unchanged (bf16).
// FP8 variant (P V too): the V tiles hold E4M3 codes of the V arena's E4M3 copy, P is stored
// as E4M3 codes of 2^6 exp2(S c - m) (four per TMEM column) with m an integer running
// reference, and P V runs as kind::f8f6f4; O and the row sum are rescaled by exact powers of
// two when the reference moves.
// Every mbarrier wait is bounded (%globaltimer); on expiry the CTA records
// FK_ERR_TIMEOUT in the status word, drains its own TMA loads and MMAs and frees TMEM.
// The kernel is launched with programmatic dependent launch: its setup (barriers, TMEM) may
// overlap the tail of the kernel before it in the stream (the compaction or current-chunk
// kernel, which write the K/V views, or whatever kernel produced Q), and the TMA thread waits
// for that kernel (griddepcontrol.wait) before its first load; every global write of this
// kernel follows MMAs that consume those loads.  It never triggers its own dependents early.
#include "fk_internal.h"

namespace fk {
namespace {

constexpr uint64_t kWaitLimitNs = 2000000000ull;   // 2 s per wait
constexpr float kRescaleThreshold = 8.0f;          // log2 units: rescale O when max grows > 2^8
// FP8 P V: P is stored as e4m3 of 2^6 exp2(s c - m), m an integer running reference (the
// running max rounded up) that lags the row max by at most 2 (rescale threshold), so P stays
// within 2^8 < 448; reference changes rescale O and l by exact powers of two
constexpr float kRescaleThresholdFp8 = 2.0f;
constexpr float kPShiftFp8 = 6.0f;

constexpr int kWarpTma = 8;                        // warps 0-3 / 4-7: softmax of query tile 0 / 1
constexpr int kWarpMma = 9;
constexpr int kAttnThreads = 320;

struct AttnBarriers {
  uint64_t q_full;
  uint64_t k_full[2], k_empty[2];   // profiling: the key ring
  uint64_t k0_full, k0_empty;       // attention: key tile 0 (stage 0)
  uint64_t vk_full[2], vk_empty[2]; // attention, b = j mod 2: V_j (V stage b) with K_{j+1} (K stage 1-b)
  uint64_t s_full[2], p_full[2];
  uint64_t o_done, fin;
  uint64_t q8_ready;            // FP8_QK: the 256 softmax threads have written the E4M3 Q rows
  uint32_t tmem_base;
  volatile int abort;
};

template <int D, bool kFp8 = false, bool kFp8PV = false>
struct Layout {
  static constexpr int kQ = kAttnBM * D * (kFp8 ? 1 : 2);   // one 128-row query tile (MMA operand)
  static constexpr int kK = kAttnBN * D * (kFp8 ? 1 : 2);   // one 128-key K tile
  static constexpr int kKV = kAttnBN * D * (kFp8PV ? 1 : 2);  // one 128-key V tile
  static constexpr int kQ16 = kFp8 ? kAttnBM * D * 2 : 0;   // FP8: one bf16 query tile as loaded
  static constexpr int kOffQ = 0;                 // two query tiles
  static constexpr int kOffK = kOffQ + 2 * kQ;    // two K stages
  static constexpr int kOffV = kOffK + 2 * kK;    // two V stages
  static constexpr int kOffQ16 = kOffV + 2 * kKV; // FP8: two bf16 query tiles
  static constexpr int kOffBar = kOffQ16 + 2 * kQ16;
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

// Non-blocking test of the phase of parity `parity` (acquire when it has completed).
__device__ __forceinline__ bool mbar_peek(uint64_t* b, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok) : "r"(su32(b)), "r"(parity) : "memory");
  return ok != 0;
}

// Bounded wait for the phase of parity `parity`.  Returns false when the CTA is
// aborting or the limit expired (which starts the abort).  Inlined: a call would save and
// restore the caller's live registers on every wait, even when the phase is complete.
__device__ __forceinline__ bool wait_phase(uint64_t* b, uint32_t parity, AttnBarriers* bar,
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
// Instruction descriptor, kind::f8f6f4: f32 accumulate, A and B E4M3 (type code 0 at bits
// 7 and 10), A K-major, B K-major (b_mn = 0) or MN-major (b_mn = 1).
__host__ __device__ constexpr uint32_t idesc_e4m3(int M, int N, int b_mn = 0) {
  return (1u << 4) | ((uint32_t)b_mn << 16) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

__device__ __forceinline__ void umma(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                     uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n"
      :: "r"(d_tmem), "l"(a), "l"(b), "r"(idesc), "r"(accumulate) : "memory");
}
// D[tmem] (+)= A[tmem] * B[smem]: A (M x 16, bf16 pairs packed along 8 columns) in tensor memory
__device__ __forceinline__ void umma_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b, uint32_t idesc,
                                        uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}\n"
      :: "r"(d_tmem), "r"(a_tmem), "l"(b), "r"(idesc), "r"(accumulate) : "memory");
}
// D[tmem] (+)= A[smem] * B[smem]^T on E4M3 operands (both K-major, K = 32 per instruction)
__device__ __forceinline__ void umma_f8(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                        uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n}\n"
      :: "r"(d_tmem), "l"(a), "l"(b), "r"(idesc), "r"(accumulate) : "memory");
}
// D[tmem] (+)= A[tmem] * B[smem] on E4M3 operands: A (M x 32, four codes per 32-bit column) in
// tensor memory, B from a shared-memory descriptor
__device__ __forceinline__ void umma_ts_f8(uint32_t d_tmem, uint32_t a_tmem, uint64_t b, uint32_t idesc,
                                           uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], [%1], %2, %3, p;\n}\n"
      :: "r"(d_tmem), "r"(a_tmem), "l"(b), "r"(idesc), "r"(accumulate) : "memory");
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

#define FK_TMEM_LD64(taddr, v)                                                              \
  asm volatile(                                                                             \
      "tcgen05.ld.sync.aligned.32x32b.x64.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,"  \
      "%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32,%33," \
      "%34,%35,%36,%37,%38,%39,%40,%41,%42,%43,%44,%45,%46,%47,%48,%49,%50,%51,%52,%53,%54," \
      "%55,%56,%57,%58,%59,%60,%61,%62,%63}, [%64];"                                        \
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),  \
        "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]),           \
        "=r"(v[13]), "=r"(v[14]), "=r"(v[15]), "=r"(v[16]), "=r"(v[17]), "=r"(v[18]),        \
        "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]),        \
        "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]),        \
        "=r"(v[31]), "=r"(v[32]), "=r"(v[33]), "=r"(v[34]), "=r"(v[35]), "=r"(v[36]),        \
        "=r"(v[37]), "=r"(v[38]), "=r"(v[39]), "=r"(v[40]), "=r"(v[41]), "=r"(v[42]),        \
        "=r"(v[43]), "=r"(v[44]), "=r"(v[45]), "=r"(v[46]), "=r"(v[47]), "=r"(v[48]),        \
        "=r"(v[49]), "=r"(v[50]), "=r"(v[51]), "=r"(v[52]), "=r"(v[53]), "=r"(v[54]),        \
        "=r"(v[55]), "=r"(v[56]), "=r"(v[57]), "=r"(v[58]), "=r"(v[59]), "=r"(v[60]),        \
        "=r"(v[61]), "=r"(v[62]), "=r"(v[63])                                               \
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

#define FK_TMEM_LD16(taddr, v)                                                              \
  asm volatile(                                                                             \
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,"  \
      "%13,%14,%15}, [%16];"                                                                \
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),  \
        "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]),           \
        "=r"(v[13]), "=r"(v[14]), "=r"(v[15])                                               \
      : "r"(taddr))

#define FK_TMEM_ST16(taddr, v)                                                              \
  asm volatile(                                                                             \
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,"   \
      "%12,%13,%14,%15,%16};"                                                               \
      :: "r"(taddr), "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]),      \
        "r"(v[6]), "r"(v[7]), "r"(v[8]), "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]),      \
        "r"(v[13]), "r"(v[14]), "r"(v[15]) : "memory")

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

// packed fp32 pair arithmetic (sm_100+): two lanes of work per instruction
__device__ __forceinline__ float2 ffma2(float2 a, float2 b, float2 c) {
  float2 d;
  asm("{\n .reg .b64 ra, rb, rc, rd;\n mov.b64 ra, {%2, %3};\n mov.b64 rb, {%4, %5};\n"
      " mov.b64 rc, {%6, %7};\n fma.rn.f32x2 rd, ra, rb, rc;\n mov.b64 {%0, %1}, rd;\n}"
      : "=f"(d.x), "=f"(d.y) : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
  return d;
}
__device__ __forceinline__ float2 fadd2(float2 a, float2 b) {
  float2 d;
  asm("{\n .reg .b64 ra, rb, rd;\n mov.b64 ra, {%2, %3};\n mov.b64 rb, {%4, %5};\n"
      " add.rn.f32x2 rd, ra, rb;\n mov.b64 {%0, %1}, rd;\n}"
      : "=f"(d.x), "=f"(d.y) : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return d;
}

// four e4m3 codes (one TMEM column of P, lowest key in the low byte) times alpha, re-rounded
__device__ __forceinline__ uint32_t scale_e4m3x4(uint32_t w, float alpha) {
  uint32_t lo, hi;
  asm("{\n .reg .b16 a, b;\n mov.b32 {a, b}, %2;\n cvt.rn.f16x2.e4m3x2 %0, a;\n"
      " cvt.rn.f16x2.e4m3x2 %1, b;\n}" : "=r"(lo), "=r"(hi) : "r"(w));
  const float2 f0 = __half22float2(*reinterpret_cast<const __half2*>(&lo));
  const float2 f1 = __half22float2(*reinterpret_cast<const __half2*>(&hi));
  return e4m3x2(f0.x * alpha, f0.y * alpha) | (e4m3x2(f1.x * alpha, f1.y * alpha) << 16);
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  const __nv_bfloat162 p = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&p);
}

// kSplit: a launch with key splits (kv_splits > 1); the unsplit instantiation carries none of
// the split bookkeeping.  kFp8: Q K^T on E4M3 operands (D = 128).  kFp8PV (with kFp8): P V on
// E4M3 operands too: V tiles from the E4M3 copy of the V view arena (one 128-byte swizzle atom
// per key row), P written as e4m3 of 2^6 exp2(s c - m), four keys per TMEM column.
template <int D, bool kSplit, bool kFp8, bool kFp8PV = false>
__global__ void __launch_bounds__(kAttnThreads, 1)
attn_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
            const __grid_constant__ CUtensorMap tmV, const AttnArgs a) {
  static_assert(!kFp8 || D == 128, "FP8_QK: one 128-byte swizzle atom per Q / K row");
  static_assert(!kFp8PV || kFp8, "FP8 P V comes with FP8 Q K^T");
  using Lay = Layout<D, kFp8, kFp8PV>;
  constexpr float kThr = kFp8PV ? kRescaleThresholdFp8 : kRescaleThreshold;
  constexpr float kPShift = kFp8PV ? kPShiftFp8 : 0.0f;
  constexpr int kHalves = D / 64;                 // 64-column (128-byte) swizzle atoms
  constexpr uint32_t kTmemCols = 512;
  constexpr uint32_t kColO = 2 * kAttnBN;         // S0 = cols 0..127, S1 = 128..255, O0, O1 after
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* sQ = smem + Lay::kOffQ;
  uint8_t* sK = smem + Lay::kOffK;
  uint8_t* sV = smem + Lay::kOffV;
  uint8_t* sQ16 = smem + Lay::kOffQ16;            // FP8: bf16 query tiles (TMA destination)
  AttnBarriers* bar = reinterpret_cast<AttnBarriers*>(smem + Lay::kOffBar);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // CTA = (head slot, pair of query tiles, key split).  Split `split` of kv_splits covers key
  // tiles [j0, j1) of the head: the CTA sees it as a head of nk keys starting at row0.
  const int split = kSplit ? blockIdx.x % a.kv_splits : 0;
  const int rest = kSplit ? blockIdx.x / a.kv_splits : blockIdx.x;
  const int hi = rest / a.n_qtiles;
  const int q0 = (rest - hi * a.n_qtiles) * (2 * kAttnBM);
  const int head = a.head_of[hi];
  int nk = a.n_keys[head];
  int row0 = a.row_base[head];
  if constexpr (kSplit) {
    const int nt_head = (nk + kAttnBN - 1) / kAttnBN;
    const int j0 = split * nt_head / a.kv_splits, j1 = (split + 1) * nt_head / a.kv_splits;
    nk = min(nk, j1 * kAttnBN) - j0 * kAttnBN;
    row0 += j0 * kAttnBN;
  }
  const int nt = (nk + kAttnBN - 1) / kAttnBN;

  if (threadIdx.x == 0) {
    mbar_init(&bar->q_full, 1);
    mbar_init(&bar->k0_full, 1);
    mbar_init(&bar->k0_empty, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bar->vk_full[i], 1);
      mbar_init(&bar->vk_empty[i], 1);
      mbar_init(&bar->s_full[i], 1);
      mbar_init(&bar->p_full[i], 4);
    }
    mbar_init(&bar->o_done, 1);
    mbar_init(&bar->fin, 1);
    if (kFp8) mbar_init(&bar->q8_ready, 2 * kAttnBM);
    bar->abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == kWarpMma) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;"
                 :: "r"(su32(&bar->tmem_base)), "r"(kTmemCols) : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bar->tmem_base;

  if (warp == kWarpTma) {
    // ------------------------------------------------------------------ TMA producer
    if (lane == 0) {
      int lastVK[2] = {-1, -1};
      bool ok = true, k0 = false;
      // Q, K and V may have been written by the previous kernel of the stream
      asm volatile("griddepcontrol.wait;" ::: "memory");
      // bf16 query tiles: the MMA operand, or (FP8) the softmax threads' quantization input
      uint8_t* q_dst = kFp8 ? sQ16 : sQ;
      constexpr int kQBytes = kAttnBM * D * 2;
      mbar_expect_tx(&bar->q_full, 2 * kQBytes);
      for (int t = 0; t < 2; ++t)
        for (int h = 0; h < kHalves; ++h)
          tma_load_3d(q_dst + t * kQBytes + h * 16384, &tmQ, &bar->q_full, h * 64, head,
                      q0 + t * kAttnBM);
      auto load_k = [&](int j, uint64_t* b) {         // key tile j into K stage j mod 2
        const int st = j & 1;
        if constexpr (kFp8) {
          tma_load_2d(sK + st * Lay::kK, &tmK, b, 0, row0 + j * kAttnBN);
        } else {
          for (int h = 0; h < kHalves; ++h)
            tma_load_2d(sK + st * Lay::kK + h * 16384, &tmK, b, h * 64, row0 + j * kAttnBN);
        }
      };
      mbar_expect_tx(&bar->k0_full, Lay::kK);
      load_k(0, &bar->k0_full);
      k0 = true;
      // then per key tile j: V_j together with K_{j+1} on one barrier (b = j mod 2).  Their
      // stages were last used by V_{j-2} and K_{j-1}, released together by vk_empty[b] after
      // iteration j-2's MMAs (K_2 reuses K_0's stage: k0_empty)
      for (int j = 0; j < nt && ok; ++j) {
        const int bb = j & 1, u = j >> 1;
        const bool more = j + 1 < nt;
        if (j >= 2 && !wait_phase(&bar->vk_empty[bb], (u - 1) & 1, bar, a.status)) { ok = false; break; }
        if (j == 1 && more && !wait_phase(&bar->k0_empty, 0, bar, a.status)) { ok = false; break; }
        mbar_expect_tx(&bar->vk_full[bb], Lay::kKV + (more ? Lay::kK : 0));
        if constexpr (kFp8PV) {
          tma_load_2d(sV + bb * Lay::kKV, &tmV, &bar->vk_full[bb], 0, row0 + j * kAttnBN);
        } else {
          for (int h = 0; h < kHalves; ++h)
            tma_load_2d(sV + bb * Lay::kKV + h * 16384, &tmV, &bar->vk_full[bb], h * 64,
                        row0 + j * kAttnBN);
        }
        if (more) load_k(j + 1, &bar->vk_full[bb]);
        lastVK[bb] = u;
      }
      if (!ok) {   // drain every load this thread issued before the CTA exits
        wait_phase(&bar->q_full, 0, bar, a.status, false);
        if (k0) wait_phase(&bar->k0_full, 0, bar, a.status, false);
        for (int bb = 0; bb < 2; ++bb)
          if (lastVK[bb] >= 0) wait_phase(&bar->vk_full[bb], lastVK[bb] & 1, bar, a.status, false);
      }
    }
    __syncwarp();
  } else if (warp == kWarpMma) {
    // ------------------------------------------------------------------ MMA issuer
    // Order per key tile j:  PV0(j), S0(j+1), PV1(j), S1(j+1).  Tensor-core operations of
    // one thread complete in issue order, so when S_t(j+1) is reported complete, PV_t(j)
    // is complete too: the softmax of tile j+1 may rescale O_t without a further wait, and
    // S_t(j+1) overwriting P_t(j) (same columns) happens after PV_t(j) has read it.
    if (lane == 0) {
      constexpr uint32_t kIdQK = kFp8 ? idesc_e4m3(kAttnBM, kAttnBN) : idesc_bf16(kAttnBM, kAttnBN, 0);
      constexpr uint32_t kIdPV = kFp8PV ? idesc_e4m3(kAttnBM, D, 1) : idesc_bf16(kAttnBM, D, 1);
      const uint32_t aQ = su32(sQ), aK = su32(sK), aV = su32(sV);
      auto qk = [&](int j, int t) {
        const int st = j & 1;
        if constexpr (kFp8) {
          // 128 codes per row = one swizzle atom: four K = 32 steps of 32 bytes
#pragma unroll
          for (int kk = 0; kk < 4; ++kk) {
            const uint64_t da = sdesc(aQ + t * Lay::kQ + kk * 32, 16, 1024);
            const uint64_t db = sdesc(aK + st * Lay::kK + kk * 32, 16, 1024);
            umma_f8(tmem + (uint32_t)(t * kAttnBN), da, db, kIdQK, kk > 0 ? 1u : 0u);
          }
        } else {
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint64_t da = sdesc(aQ + t * Lay::kQ + (kk >> 2) * 16384 + (kk & 3) * 32, 16, 1024);
            const uint64_t db = sdesc(aK + st * Lay::kK + (kk >> 2) * 16384 + (kk & 3) * 32, 16, 1024);
            umma(tmem + (uint32_t)(t * kAttnBN), da, db, kIdQK, kk > 0 ? 1u : 0u);
          }
        }
        umma_commit(&bar->s_full[t]);
      };
      auto pv = [&](int j, int t) {
        const int st = j & 1;
        if constexpr (kFp8PV) {
          // 32 keys per step: P columns 8 kk .. 8 kk + 7 (four codes each); V rows 32 kk .. +31,
          // MN-major (d contiguous, 128 bytes per key row), 8-row groups 1024 bytes apart
#pragma unroll
          for (int kk = 0; kk < kAttnBN / 32; ++kk) {
            const uint64_t db = sdesc(aV + st * Lay::kKV + kk * 4096, 16384, 1024);
            umma_ts_f8(tmem + kColO + (uint32_t)(t * D), tmem + (uint32_t)(t * kAttnBN + kk * 8), db,
                       kIdPV, (j > 0 || kk > 0) ? 1u : 0u);
          }
        } else {
#pragma unroll
          for (int kk = 0; kk < kAttnBN / 16; ++kk) {
            const uint64_t db = sdesc(aV + st * Lay::kKV + kk * 2048, 16384, 1024);
            umma_ts(tmem + kColO + (uint32_t)(t * D), tmem + (uint32_t)(t * kAttnBN + kk * 8), db,
                    kIdPV, (j > 0 || kk > 0) ? 1u : 0u);
          }
        }
      };
      bool ok = wait_phase(kFp8 ? &bar->q8_ready : &bar->q_full, 0, bar, a.status) &&
                wait_phase(&bar->k0_full, 0, bar, a.status);
      if (ok) {
        tc_fence_after();
        qk(0, 0);
        qk(0, 1);
        umma_commit(&bar->k0_empty);
      }
      // barriers found complete by a test made while the pipe was busy with the group just issued
      // need no wait afterwards (each wait costs ~100 cycles where the pipe would drain)
      bool vk_ready = false;
      for (int j = 0; j < nt && ok; ++j) {
        const int bb = j & 1;
        const bool more = j + 1 < nt;
        // V_j and K_{j+1} (one barrier) before P_0(j): neither depends on the softmax, and
        // PV0(j), S0(j+1) then go to the tensor pipe back to back once P_0(j) is in TMEM
        if (!(vk_ready || wait_phase(&bar->vk_full[bb], (j >> 1) & 1, bar, a.status)) ||
            !wait_phase(&bar->p_full[0], j & 1, bar, a.status)) { ok = false; break; }
        tc_fence_after();
        pv(j, 0);
        const bool p1_ready = mbar_peek(&bar->p_full[1], j & 1);
        if (more) qk(j + 1, 0);
        if (!(p1_ready || wait_phase(&bar->p_full[1], j & 1, bar, a.status))) { ok = false; break; }
        tc_fence_after();
        pv(j, 1);
        vk_ready = more && mbar_peek(&bar->vk_full[(j + 1) & 1], ((j + 1) >> 1) & 1);
        if (more) qk(j + 1, 1);
        umma_commit(&bar->vk_empty[bb]);             // V_j and K_{j+1} consumed
      }
      if (ok) umma_commit(&bar->o_done);
      umma_commit(&bar->fin);                       // completes once every MMA above is done
      wait_phase(&bar->fin, 0, bar, a.status, false);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------------ softmax warpgroups
    const int t = warp >> 2;                        // query tile of this warpgroup
    const int wq = warp & 3;
    const int row = wq * 32 + lane;
    const uint32_t lane_base = (uint32_t)(wq * 32) << 16;
    const uint32_t tS = tmem + lane_base + (uint32_t)(t * kAttnBN);
    const uint32_t tO = tmem + lane_base + kColO + (uint32_t)(t * D);
    // logit scale of this row in the log2 domain: log2(e) / sqrt(D), times 2^e_row for E4M3
    // queries (e_row in [-120, 120]: the product is exact)
    float sl2 = a.scale_log2;
    bool ok = true;
    if constexpr (kFp8) {
      // quantize this thread's query row: the bf16 row (two 64-element swizzle atoms, 16-byte
      // chunk j of row r at chunk j ^ (r & 7)) -> max |q| -> e -> E4M3 codes of q 2^-e, 128 bytes
      // in the same swizzle pattern (rows past Nq were zero-filled: e = 0, codes 0)
      if (warp_wait(&bar->q_full, 0, bar, a.status)) {
        const uint8_t* src = sQ16 + t * (kAttnBM * D * 2) + row * 128;
        uint4 v[16];
#pragma unroll
        for (int j = 0; j < 16; ++j)
          v[j] = *reinterpret_cast<const uint4*>(src + (j >> 3) * 16384 + (((j & 7) ^ (row & 7)) << 4));
        float amax = 0.0f;
#pragma unroll
        for (int j = 0; j < 16; ++j) amax = fmaxf(amax, absmax8(v[j]));
        const int e = e4m3_row_exponent(amax);
        const float inv = pow2f(-e);
        uint8_t* dst = sQ + t * Lay::kQ + row * 128;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const uint2 lo = e4m3x8(v[2 * j], inv), hi = e4m3x8(v[2 * j + 1], inv);
          *reinterpret_cast<uint4*>(dst + ((j ^ (row & 7)) << 4)) = make_uint4(lo.x, lo.y, hi.x, hi.y);
        }
        sl2 *= pow2f(e);
        // the tensor core reads shared memory through the async proxy
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      } else {
        ok = false;
      }
      mbar_arrive(&bar->q8_ready);
    }
    float m = -INFINITY, l = 0.0f;
    for (int j = 0; j < nt && ok; ++j) {
      if (!warp_wait(&bar->s_full[t], j & 1, bar, a.status)) { ok = false; break; }
      tc_fence_after();
      const int valid = nk - j * kAttnBN;           // keys of this tile (< 128 only in the last)
      const bool full = valid >= kAttnBN;           // uniform over the CTA
      const float2 sc2 = make_float2(sl2, sl2);
      float2 acc[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) acc[i] = make_float2(0.0f, 0.0f);
      float alpha_tile = 1.0f;
      bool rescaled = false;
      // One pass per 64-column half: the half's maximum (eight independent chains), a lazy
      // update of the running max m (only when it grows by more than 2^8), then
      // P = exp2(S*c - m) as bf16 pairs written over the S columns already read (P columns
      // 32h..32h+31 come from S columns 64h..64h+63): the A operand of PV.  FP8 P V: m is the
      // running max rounded up to an integer, updated when it grows by more than 2, and P the
      // e4m3 codes of 2^6 exp2(S*c - m), four per column (P columns 16h..16h+15).  If the second
      // half raises m, the first half's stored P is rescaled in place.
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        uint32_t sv[64];
        FK_TMEM_LD64(tS + half * 64, sv);
        tmem_wait_ld();
        if constexpr (!kFp8PV) {
          // Full tile after the first (every row has a finite running max m): P = exp2(S*c - m)
          // straight away; m has to move only if some P exceeds 2^8 (an element more than 8
          // above m), which the packed bf16 maximum of the half's P shows.  Otherwise the
          // half is done without a separate max pass; if it does, the path below redoes it.
          if (full && j > 0) {
            uint32_t pk[32];
            float2 ah[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) ah[i] = make_float2(0.0f, 0.0f);
            const float2 nm2 = make_float2(-m, -m);
#pragma unroll
            for (int q = 0; q < 32; ++q) {
              const float2 x = ffma2(make_float2(__uint_as_float(sv[2 * q]), __uint_as_float(sv[2 * q + 1])),
                                     sc2, nm2);
              float2 e;
              e.x = fast_exp2(x.x);
              e.y = fast_exp2(x.y);
              ah[q & 3] = fadd2(ah[q & 3], e);
              pk[q] = pack_bf16(e.x, e.y);
            }
            // the half's sum bounds each of its numerators: only a sum above 2^8 needs the max
            const float2 hs2 = fadd2(fadd2(ah[0], ah[1]), fadd2(ah[2], ah[3]));
            bool over = false;
            if (__any_sync(0xffffffffu, hs2.x + hs2.y > 256.0f)) {
              __nv_bfloat162 pm[4];
#pragma unroll
              for (int i = 0; i < 4; ++i) pm[i] = *reinterpret_cast<const __nv_bfloat162*>(&pk[i]);
#pragma unroll
              for (int q = 4; q < 32; ++q)
                pm[q & 3] = __hmax2(pm[q & 3], *reinterpret_cast<const __nv_bfloat162*>(&pk[q]));
              const __nv_bfloat162 p2 = __hmax2(__hmax2(pm[0], pm[1]), __hmax2(pm[2], pm[3]));
              over = fmaxf(__low2float(p2), __high2float(p2)) > 256.0f;
            }
            if (!__any_sync(0xffffffffu, over)) {                          // warp-uniform
#pragma unroll
              for (int i = 0; i < 4; ++i) acc[i] = fadd2(acc[i], ah[i]);
              FK_TMEM_ST32(tS + half * 32, pk);
              continue;
            }
          }
        } else {
          // FP8 P V, the same idea with the integer reference: a numerator above 2^8 (y more than
          // 2 above m) shows as an e4m3 code above 0x78; codes are non-negative and at most 0x7E,
          // so adding 7 to each byte sets its top bit exactly then, without carries between bytes
          if (full && j > 0) {
            uint32_t pk[16], ov = 0;
            float2 ah[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) ah[i] = make_float2(0.0f, 0.0f);
            const float2 nm2 = make_float2(kPShift - m, kPShift - m);
#pragma unroll
            for (int q = 0; q < 16; ++q) {
              const float2 x0 = ffma2(make_float2(__uint_as_float(sv[4 * q]), __uint_as_float(sv[4 * q + 1])),
                                      sc2, nm2);
              const float2 x1 = ffma2(make_float2(__uint_as_float(sv[4 * q + 2]), __uint_as_float(sv[4 * q + 3])),
                                      sc2, nm2);
              float2 e0, e1;
              e0.x = fast_exp2(x0.x);
              e0.y = fast_exp2(x0.y);
              e1.x = fast_exp2(x1.x);
              e1.y = fast_exp2(x1.y);
              ah[(2 * q) & 3] = fadd2(ah[(2 * q) & 3], e0);
              ah[(2 * q + 1) & 3] = fadd2(ah[(2 * q + 1) & 3], e1);
              pk[q] = e4m3x2(e0.x, e0.y) | (e4m3x2(e1.x, e1.y) << 16);
              ov |= pk[q] + 0x07070707u;
            }
            if (!__any_sync(0xffffffffu, (ov & 0x80808080u) != 0)) {   // warp-uniform
#pragma unroll
              for (int i = 0; i < 4; ++i) acc[i] = fadd2(acc[i], ah[i]);
              FK_TMEM_ST16(tS + half * 16, pk);
              continue;
            }
          }
        }
        float mxa[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) mxa[i] = -INFINITY;
        if (full) {
#pragma unroll
          for (int c = 0; c < 64; ++c) mxa[c & 7] = fmaxf(mxa[c & 7], __uint_as_float(sv[c]));
        } else {
#pragma unroll
          for (int c = 0; c < 64; ++c)
            if (half * 64 + c < valid) mxa[c & 7] = fmaxf(mxa[c & 7], __uint_as_float(sv[c]));
        }
        const float mx = fmaxf(fmaxf(fmaxf(mxa[0], mxa[1]), fmaxf(mxa[2], mxa[3])),
                               fmaxf(fmaxf(mxa[4], mxa[5]), fmaxf(mxa[6], mxa[7])));
        const float m_new = fmaxf(m, kFp8PV ? ceilf(mx * sl2) : mx * sl2);
        if (__any_sync(0xffffffffu, m_new > m + kThr)) {               // warp-uniform
          float alpha;                               // 0 when m = -inf
          if constexpr (kFp8PV) {                    // integer references: an exact power of two
            const float dm = m - m_new;
            alpha = (m == -INFINITY || dm < -126.0f) ? 0.0f : pow2f((int)dm);
          } else {
            alpha = fast_exp2(m - m_new);
          }
          l *= alpha;
#pragma unroll
          for (int i = 0; i < 4; ++i) acc[i] = make_float2(acc[i].x * alpha, acc[i].y * alpha);
          if (half == 1) {                           // rare: first half of P was stored with the old m
            if constexpr (kFp8PV) {
              uint32_t p0[16];
              tmem_wait_st();
              FK_TMEM_LD16(tS, p0);
              tmem_wait_ld();
#pragma unroll
              for (int e = 0; e < 16; ++e) p0[e] = scale_e4m3x4(p0[e], alpha);
              FK_TMEM_ST16(tS, p0);
            } else {
              uint32_t p0[32];
              tmem_wait_st();
              FK_TMEM_LD32(tS, p0);
              tmem_wait_ld();
#pragma unroll
              for (int e = 0; e < 32; ++e) {
                const __nv_bfloat162 b = *reinterpret_cast<const __nv_bfloat162*>(&p0[e]);
                p0[e] = pack_bf16(__low2float(b) * alpha, __high2float(b) * alpha);
              }
              FK_TMEM_ST32(tS, p0);
            }
          }
          alpha_tile *= alpha;
          rescaled = true;
          m = m_new;
        }
        const float2 nm2 = make_float2(kPShift - m, kPShift - m);
        if constexpr (kFp8PV) {
          uint32_t pk[16];
          if (!full) {                               // the ragged last tile: masked keys give 0
#pragma unroll
            for (int c = 0; c < 64; ++c)
              if (half * 64 + c >= valid) sv[c] = __float_as_uint(-INFINITY);
          }
#pragma unroll
          for (int q = 0; q < 16; ++q) {
            const float2 x0 = ffma2(make_float2(__uint_as_float(sv[4 * q]), __uint_as_float(sv[4 * q + 1])),
                                    sc2, nm2);
            const float2 x1 = ffma2(make_float2(__uint_as_float(sv[4 * q + 2]), __uint_as_float(sv[4 * q + 3])),
                                    sc2, nm2);
            float2 e0, e1;
            e0.x = fast_exp2(x0.x);
            e0.y = fast_exp2(x0.y);
            e1.x = fast_exp2(x1.x);
            e1.y = fast_exp2(x1.y);
            acc[(2 * q) & 3] = fadd2(acc[(2 * q) & 3], e0);
            acc[(2 * q + 1) & 3] = fadd2(acc[(2 * q + 1) & 3], e1);
            pk[q] = e4m3x2(e0.x, e0.y) | (e4m3x2(e1.x, e1.y) << 16);
          }
          FK_TMEM_ST16(tS + half * 16, pk);
          continue;
        }
        uint32_t pk[32];
        if (full) {
#pragma unroll
          for (int q = 0; q < 32; ++q) {
            const float2 x = ffma2(make_float2(__uint_as_float(sv[2 * q]), __uint_as_float(sv[2 * q + 1])),
                                   sc2, nm2);
            float2 e;
            e.x = fast_exp2(x.x);                    // MUFU
            e.y = fast_exp2(x.y);
            acc[q & 3] = fadd2(acc[q & 3], e);
            pk[q] = pack_bf16(e.x, e.y);
          }
        } else {
#pragma unroll
          for (int q = 0; q < 32; ++q) {
            const int c = half * 64 + 2 * q;
            const float x0 = c < valid ? __uint_as_float(sv[2 * q]) : -INFINITY;
            const float x1 = c + 1 < valid ? __uint_as_float(sv[2 * q + 1]) : -INFINITY;
            float2 e;
            e.x = fast_exp2(fmaf(x0, sl2, -m));
            e.y = fast_exp2(fmaf(x1, sl2, -m));
            acc[q & 3] = fadd2(acc[q & 3], e);
            pk[q] = pack_bf16(e.x, e.y);
          }
        }
        FK_TMEM_ST32(tS + half * 32, pk);
      }
      const float2 acc01 = fadd2(acc[0], acc[1]), acc23 = fadd2(acc[2], acc[3]);
      const float2 acc4 = fadd2(acc01, acc23);
      l += acc4.x + acc4.y;
      if (rescaled && j > 0) {                       // PV_t(j-1) is complete (see MMA order)
#pragma unroll
        for (int c = 0; c < D / 32; ++c) {
          uint32_t o[32];
          FK_TMEM_LD32(tO + c * 32, o);
          tmem_wait_ld();
#pragma unroll
          for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha_tile);
          FK_TMEM_ST32(tO + c * 32, o);
        }
      }
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bar->p_full[t]);
    }
    // ---------------------------------------------------------------- epilogue
    if (kSplit && ok && warp_wait(&bar->o_done, 0, bar, a.status)) {
      // one key split: unnormalised O and the row's (m, l), merged by merge_kernel
      tc_fence_after();
      const int q = q0 + t * kAttnBM + row;
      const int64_t slot = ((int64_t)split * a.Nq + q) * a.H + head;
      float* prow = a.part_o + slot * D;
#pragma unroll
      for (int c = 0; c < D / 32; ++c) {
        uint32_t o[32];
        FK_TMEM_LD32(tO + c * 32, o);
        tmem_wait_ld();
        if (q < a.Nq) {
#pragma unroll
          for (int e = 0; e < 32; e += 4)
            *reinterpret_cast<uint4*>(prow + c * 32 + e) = make_uint4(o[e], o[e + 1], o[e + 2], o[e + 3]);
        }
      }
      if (q < a.Nq) a.part_ml[slot] = make_float2(m, l);
    } else if (!kSplit && ok && warp_wait(&bar->o_done, 0, bar, a.status)) {
      tc_fence_after();
      const float inv = 1.0f / l;
      const int q = q0 + t * kAttnBM + row;
      bf16* orow = a.O + ((int64_t)q * a.H + head) * D;
#pragma unroll
      for (int c = 0; c < D / 32; ++c) {
        uint32_t o[32];
        FK_TMEM_LD32(tO + c * 32, o);
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
  if (warp == kWarpMma) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" :: "r"(tmem),
                 "r"(kTmemCols) : "memory");
  }
}

// ---------------------------------------------------------------------------------------
// Offline head profiling (Sec. 4.1, Eq. 1): per head, the attention mass that the queries of
// the generated chunk put on the generated chunk, the transition (anchor) frame and the sink
// frames, out of a full softmax over every key of the attention window.  Keys are ordered
// [generated | sink | other history | transition].  S = Q K^T runs on the tensor cores
// (tcgen05, S double-buffered in 256 TMEM columns); no P V product is needed.  Per row the
// softmax statistics are kept online (running max, total sum, and the three class sums,
// rescaled together); the per-row fractions are summed per head in double.  A cluster of two
// CTAs handles one (head, 128-row query tile), each CTA half of the key tiles (so the grid
// fills the SMs in about three even waves instead of two, the second half empty); the
// second CTA writes its row statistics into the first's shared memory (distributed shared
// memory, one cluster barrier), and the first merges the two ranges.
//   warps 0-3  statistics of rows 0..127 (TMEM lanes), one thread per row;
//   warp 4     TMA: the query tile once, key tiles into a two-stage ring;
//   warp 5     tcgen05.mma: S_b = Q K_j^T for b = j mod 2, once the statistics warps have
//              read S_b of tile j - 2 (they release it right after their TMEM loads).
constexpr int kProfThreads = 192;
constexpr int kWarpProfTma = 4;
constexpr int kWarpProfMma = 5;

template <int D>
struct ProfLayout {
  static constexpr int kQ = kAttnBM * D * 2;
  static constexpr int kK = kAttnBN * D * 2;
  static constexpr int kOffQ = 0;
  static constexpr int kOffK = kOffQ + kQ;
  static constexpr int kOffBar = kOffK + 2 * kK;
  static constexpr int kOffPart = kOffBar + 256;      // the cluster peer's row statistics
  static constexpr int kSmem = kOffPart + kAttnBM * 8 * 4 + 1024;   // + alignment slack; two CTAs per SM
};

template <int D>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kProfThreads, 2)
profile_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
               const ProfArgs a) {
  using Lay = ProfLayout<D>;
  constexpr int kHalves = D / 64;
  constexpr uint32_t kTmemCols = 256;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* sQ = smem + Lay::kOffQ;
  uint8_t* sK = smem + Lay::kOffK;
  AttnBarriers* bar = reinterpret_cast<AttnBarriers*>(smem + Lay::kOffBar);
  // barrier use: q_full, k_full/k_empty (key ring), s_full[b] (S_b written), p_full[b]
  // (S_b read by the four statistics warps), fin

  float* part = reinterpret_cast<float*>(smem + Lay::kOffPart);   // [row][8]: m l cg cs ct ok
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int row = warp * 32 + lane;                 // query row of a statistics thread
  // A cluster of two CTAs = one (head, query tile); CTA r of the cluster takes key tiles
  // [j0, j0 + nt) of the head's window (r = 0 the first half, r = 1 the rest).
  uint32_t rank;
  asm("mov.u32 %0, %%cluster_ctarank;" : "=r"(rank));
  const int pair = blockIdx.x >> 1;
  const int head = pair / a.n_qtiles;
  const int q0 = (pair - head * a.n_qtiles) * kAttnBM;
  const int nk = a.Nk;
  const int nt_all = (nk + kAttnBN - 1) / kAttnBN;
  const int j0 = rank ? nt_all / 2 : 0;
  const int nt = rank ? nt_all - nt_all / 2 : nt_all / 2;   // may be 0 (one key tile in all)
  // row statistics of this CTA's keys (statistics warps): running max (log2 domain), total
  // sum and the class sums, all relative to m
  float m = -INFINITY, l = 0.0f, cg = 0.0f, cs = 0.0f, ct = 0.0f;
  bool ok = true;

  if (threadIdx.x == 0) {
    mbar_init(&bar->q_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bar->k_full[i], 1);
      mbar_init(&bar->k_empty[i], 1);
      mbar_init(&bar->s_full[i], 1);
      mbar_init(&bar->p_full[i], 4);
    }
    mbar_init(&bar->fin, 1);
    bar->abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == kWarpProfMma) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;"
                 :: "r"(su32(&bar->tmem_base)), "r"(kTmemCols) : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bar->tmem_base;

  if (warp == kWarpProfTma) {
    if (lane == 0) {
      int lastK[2] = {-1, -1};
      bool ok = true;
      mbar_expect_tx(&bar->q_full, Lay::kQ);
      for (int h = 0; h < kHalves; ++h)
        tma_load_3d(sQ + h * 16384, &tmQ, &bar->q_full, h * 64, head, q0);
      for (int j = 0; j < nt; ++j) {
        const int st = j & 1, u = j >> 1;
        if (j >= 2 && !wait_phase(&bar->k_empty[st], (u - 1) & 1, bar, a.status)) { ok = false; break; }
        mbar_expect_tx(&bar->k_full[st], Lay::kK);
        for (int h = 0; h < kHalves; ++h)
          tma_load_3d(sK + st * Lay::kK + h * 16384, &tmK, &bar->k_full[st], h * 64, head,
                      (j0 + j) * kAttnBN);
        lastK[st] = u;
      }
      if (!ok) {   // drain every load this thread issued before the CTA exits
        wait_phase(&bar->q_full, 0, bar, a.status, false);
        for (int st = 0; st < 2; ++st)
          if (lastK[st] >= 0) wait_phase(&bar->k_full[st], lastK[st] & 1, bar, a.status, false);
      }
    }
    __syncwarp();
  } else if (warp == kWarpProfMma) {
    if (lane == 0) {
      constexpr uint32_t kIdQK = idesc_bf16(kAttnBM, kAttnBN, 0);
      const uint32_t aQ = su32(sQ), aK = su32(sK);
      bool ok = wait_phase(&bar->q_full, 0, bar, a.status);
      for (int j = 0; j < nt && ok; ++j) {
        const int st = j & 1, u = j >> 1;
        if (!wait_phase(&bar->k_full[st], u & 1, bar, a.status) ||
            (j >= 2 && !wait_phase(&bar->p_full[st], (u - 1) & 1, bar, a.status))) { ok = false; break; }
        tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint64_t da = sdesc(aQ + (kk >> 2) * 16384 + (kk & 3) * 32, 16, 1024);
          const uint64_t db = sdesc(aK + st * Lay::kK + (kk >> 2) * 16384 + (kk & 3) * 32, 16, 1024);
          umma(tmem + (uint32_t)(st * kAttnBN), da, db, kIdQK, kk > 0 ? 1u : 0u);
        }
        umma_commit(&bar->s_full[st]);
        umma_commit(&bar->k_empty[st]);
      }
      umma_commit(&bar->fin);                       // completes once every MMA above is done
      wait_phase(&bar->fin, 0, bar, a.status, false);
    }
    __syncwarp();
  } else {
    const int wq = warp;
    const uint32_t lane_base = (uint32_t)(wq * 32) << 16;
    for (int j = 0; j < nt; ++j) {
      const int st = j & 1;
      if (!warp_wait(&bar->s_full[st], (j >> 1) & 1, bar, a.status)) { ok = false; break; }
      tc_fence_after();
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        const int kb = (j0 + j) * kAttnBN + half * 64;   // first key of this half
        const int valid = min(64, nk - kb);          // uniform over the CTA
        uint32_t sv[64];
        FK_TMEM_LD64(tmem + lane_base + (uint32_t)(st * kAttnBN + half * 64), sv);
        tmem_wait_ld();
        if (half == 1) {                             // S_b is in registers: release it
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&bar->p_full[st]);
        }
        if (valid <= 0) continue;
        // key classes are contiguous ranges in the order generated, sink, other, transition
        const int last = kb + valid - 1;
        const int cls_first = kb < a.g_end ? 0 : kb < a.s_end ? 1 : kb >= a.t_begin ? 3 : 2;
        const int cls_last = last < a.g_end ? 0 : last < a.s_end ? 1 : last >= a.t_begin ? 3 : 2;
        // A full half of one key class after the first half (every row then has a finite
        // running max m): the exponentials with m straight away.  The half's sum bounds each
        // term, so only a sum above 2^8 (possibly a key more than 8 above m in log2 units)
        // needs the max pass and lazy rescale below, which then redoes the half.
        if (valid == 64 && cls_first == cls_last && (j > 0 || half > 0)) {   // CTA-uniform
          const float2 sc2 = make_float2(a.scale_log2, a.scale_log2), nm2 = make_float2(-m, -m);
          float2 a2[4];
#pragma unroll
          for (int i = 0; i < 4; ++i) a2[i] = make_float2(0.0f, 0.0f);
#pragma unroll
          for (int q = 0; q < 32; ++q) {
            const float2 x = ffma2(make_float2(__uint_as_float(sv[2 * q]), __uint_as_float(sv[2 * q + 1])),
                                   sc2, nm2);
            a2[q & 3] = fadd2(a2[q & 3], make_float2(fast_exp2(x.x), fast_exp2(x.y)));
          }
          const float2 s2 = fadd2(fadd2(a2[0], a2[1]), fadd2(a2[2], a2[3]));
          const float sum = s2.x + s2.y;
          if (!__any_sync(0xffffffffu, sum > 256.0f)) {                  // warp-uniform
            l += sum;
            if (cls_first == 0) cg += sum;
            else if (cls_first == 1) cs += sum;
            else if (cls_first == 3) ct += sum;
            continue;
          }
        }
        float mxa[8];                                // eight independent max chains
#pragma unroll
        for (int i = 0; i < 8; ++i) mxa[i] = -INFINITY;
#pragma unroll
        for (int c = 0; c < 64; ++c)
          if (c < valid) mxa[c & 7] = fmaxf(mxa[c & 7], __uint_as_float(sv[c]));
        const float mx = fmaxf(fmaxf(fmaxf(mxa[0], mxa[1]), fmaxf(mxa[2], mxa[3])),
                               fmaxf(fmaxf(mxa[4], mxa[5]), fmaxf(mxa[6], mxa[7])));
        const float m_new = fmaxf(m, mx * a.scale_log2);
        if (__any_sync(0xffffffffu, m_new > m + kRescaleThreshold)) {   // warp-uniform
          const float alpha = fast_exp2(m - m_new);  // 0 when m = -inf
          l *= alpha;
          cg *= alpha;
          cs *= alpha;
          ct *= alpha;
          m = m_new;
        }
        if (cls_first == cls_last) {
          float acc[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
          for (int c = 0; c < 64; ++c)
            if (c < valid) acc[c & 3] += fast_exp2(fmaf(__uint_as_float(sv[c]), a.scale_log2, -m));
          const float sum = (acc[0] + acc[1]) + (acc[2] + acc[3]);
          l += sum;
          if (cls_first == 0) cg += sum;
          else if (cls_first == 1) cs += sum;
          else if (cls_first == 3) ct += sum;
        } else {
#pragma unroll
          for (int c = 0; c < 64; ++c) {
            if (c < valid) {
              const int key = kb + c;
              const float e = fast_exp2(fmaf(__uint_as_float(sv[c]), a.scale_log2, -m));
              l += e;
              if (key < a.g_end) cg += e;
              else if (key < a.s_end) cs += e;
              else if (key >= a.t_begin) ct += e;
            }
          }
        }
      }
    }
    if (rank == 1) {
      // this CTA's row statistics go to the same row slot in the first CTA's shared memory
      uint32_t dst;
      asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(dst) : "r"(su32(part + row * 8)), "r"(0u));
      asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" :: "r"(dst), "f"(m), "f"(l),
                   "f"(cg), "f"(cs) : "memory");
      asm volatile("st.shared::cluster.v2.f32 [%0], {%1, %2};" :: "r"(dst + 16u), "f"(ct),
                   "f"(ok ? 1.0f : 0.0f) : "memory");
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == kWarpProfMma) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" :: "r"(tmem),
                 "r"(kTmemCols) : "memory");
  }
  // every thread of both CTAs: the second CTA's statistics have landed (release / acquire)
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
  if (rank == 0 && warp < kWarpProfTma) {
    // merge the two key ranges: with M = max(m0, m1), every sum s = s0 2^(m0 - M) + s1 2^(m1 - M)
    const float* pp = part + row * 8;
    const float pm = pp[0];
    ok = ok && pp[5] != 0.0f;                       // warp-uniform: one warp of each CTA per row block
    const float M = fmaxf(m, pm);
    const float w0 = m == -INFINITY ? 0.0f : fast_exp2(m - M);
    const float w1 = pm == -INFINITY ? 0.0f : fast_exp2(pm - M);
    l = l * w0 + pp[1] * w1;
    cg = cg * w0 + pp[2] * w1;
    cs = cs * w0 + pp[3] * w1;
    ct = ct * w0 + pp[4] * w1;
    if (ok) {
      const bool in = q0 + row < a.Nq;
      float fg = in ? cg / l : 0.0f, fs = in ? cs / l : 0.0f, ft = in ? ct / l : 0.0f;
      float rows = in ? 1.0f : 0.0f;
#pragma unroll
      for (int sft = 16; sft >= 1; sft >>= 1) {
        fg += __shfl_xor_sync(0xffffffffu, fg, sft);
        fs += __shfl_xor_sync(0xffffffffu, fs, sft);
        ft += __shfl_xor_sync(0xffffffffu, ft, sft);
        rows += __shfl_xor_sync(0xffffffffu, rows, sft);
      }
      if (lane == 0 && rows > 0.0f) {
        double* mh = a.mass + (int64_t)head * 4;
        atomicAdd(mh + 0, (double)rows);
        atomicAdd(mh + 1, (double)fg);
        atomicAdd(mh + 2, (double)ft);
        atomicAdd(mh + 3, (double)fs);
      }
    }
  }
}

}  // namespace

cudaError_t launch_head_profile(int head_dim, const CUtensorMap& tmQ, const CUtensorMap& tmK,
                                const ProfArgs& a, cudaStream_t s) {
  const unsigned grid = (unsigned)(2 * a.n_qtiles * a.H);   // clusters of two CTAs
  cudaError_t e;
  if (head_dim == 128) {
    e = cudaFuncSetAttribute(profile_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             ProfLayout<128>::kSmem);
    if (e != cudaSuccess) return e;
    profile_kernel<128><<<grid, kProfThreads, ProfLayout<128>::kSmem, s>>>(tmQ, tmK, a);
  } else {
    e = cudaFuncSetAttribute(profile_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             ProfLayout<64>::kSmem);
    if (e != cudaSuccess) return e;
    profile_kernel<64><<<grid, kProfThreads, ProfLayout<64>::kSmem, s>>>(tmQ, tmK, a);
  }
  return cudaGetLastError();
}

namespace {

// Merge of the key splits of one query row and head (one warp): with M = max_s m_s (log2
// domain), O = sum_s 2^(m_s - M) O_s / sum_s 2^(m_s - M) l_s, stored as bf16.
template <int D>
__global__ void __launch_bounds__(256) merge_kernel(const float* part_o, const float2* part_ml,
                                                    bf16* O, int Nq, int H, int splits) {
  constexpr int kPer = D / 32;
  const int64_t w = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (w >= (int64_t)Nq * H) return;
  float M = -INFINITY;
  for (int sp = 0; sp < splits; ++sp) M = fmaxf(M, part_ml[sp * (int64_t)Nq * H + w].x);
  float L = 0.0f, acc[kPer];
#pragma unroll
  for (int d = 0; d < kPer; ++d) acc[d] = 0.0f;
  for (int sp = 0; sp < splits; ++sp) {
    const int64_t slot = sp * (int64_t)Nq * H + w;
    const float2 ml = part_ml[slot];
    const float wgt = fast_exp2(ml.x - M);
    L = fmaf(wgt, ml.y, L);
    const float* src = part_o + slot * D + lane * kPer;
#pragma unroll
    for (int d = 0; d < kPer; ++d) acc[d] = fmaf(wgt, src[d], acc[d]);
  }
  const float inv = 1.0f / L;
  bf16* dst = O + w * D + lane * kPer;
#pragma unroll
  for (int d = 0; d < kPer; d += 2)
    *reinterpret_cast<uint32_t*>(dst + d) = pack_bf16(acc[d] * inv, acc[d + 1] * inv);
}

}  // namespace

void launch_merge(int head_dim, const AttnArgs& a, cudaStream_t s) {
  const int64_t warps = (int64_t)a.Nq * a.H;
  const unsigned grid = (unsigned)((warps * 32 + 255) / 256);
  if (head_dim == 128) merge_kernel<128><<<grid, 256, 0, s>>>(a.part_o, a.part_ml, a.O, a.Nq, a.H, a.kv_splits);
  else merge_kernel<64><<<grid, 256, 0, s>>>(a.part_o, a.part_ml, a.O, a.Nq, a.H, a.kv_splits);
}

cudaError_t attention_prepare(int head_dim) {
  const auto set = [](const void* fn, int smem) {
    return cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  };
  cudaError_t e;
  if (head_dim == 128) {
    if ((e = set((const void*)attn_kernel<128, false, false>, Layout<128>::kSmem)) != cudaSuccess) return e;
    if ((e = set((const void*)attn_kernel<128, true, false>, Layout<128>::kSmem)) != cudaSuccess) return e;
    if ((e = set((const void*)attn_kernel<128, false, true>, Layout<128, true>::kSmem)) != cudaSuccess) return e;
    if ((e = set((const void*)attn_kernel<128, true, true>, Layout<128, true>::kSmem)) != cudaSuccess) return e;
    if ((e = set((const void*)attn_kernel<128, false, true, true>, Layout<128, true, true>::kSmem)) != cudaSuccess)
      return e;
    return set((const void*)attn_kernel<128, true, true, true>, Layout<128, true, true>::kSmem);
  }
  if ((e = set((const void*)attn_kernel<64, false, false>, Layout<64>::kSmem)) != cudaSuccess) return e;
  return set((const void*)attn_kernel<64, true, false>, Layout<64>::kSmem);
}

void launch_attention(int head_dim, int precision, const CUtensorMap& tmQ, const CUtensorMap& tmK,
                      const CUtensorMap& tmV, const AttnArgs& a, cudaStream_t s) {
  using Kern = void (*)(const CUtensorMap, const CUtensorMap, const CUtensorMap, const AttnArgs);
  const bool split = a.kv_splits > 1;
  Kern kern;
  int smem;
  if (head_dim == 128 && precision == FK_ATTN_FP8) {
    kern = split ? attn_kernel<128, true, true, true> : attn_kernel<128, false, true, true>;
    smem = Layout<128, true, true>::kSmem;
  } else if (head_dim == 128 && precision == FK_ATTN_FP8_QK) {
    kern = split ? attn_kernel<128, true, true> : attn_kernel<128, false, true>;
    smem = Layout<128, true>::kSmem;
  } else if (head_dim == 128) {
    kern = split ? attn_kernel<128, true, false> : attn_kernel<128, false, false>;
    smem = Layout<128>::kSmem;
  } else {
    kern = split ? attn_kernel<64, true, false> : attn_kernel<64, false, false>;
    smem = Layout<64>::kSmem;
  }
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3((unsigned)(a.n_qtiles * a.H * a.kv_splits));
  cfg.blockDim = dim3(kAttnThreads);
  cfg.dynamicSmemBytes = (size_t)smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaLaunchKernelEx(&cfg, kern, tmQ, tmK, tmV, a);
}

}  // namespace fk
