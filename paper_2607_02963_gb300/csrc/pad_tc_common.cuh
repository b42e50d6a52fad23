// Device helpers shared by the tensor-core kernels of the prefix pass (pad_prefix_tc.cu,
// pad_prefix_dual.cu): mbarriers with bounded waits, TMA tile loads, tcgen05 MMA / TMEM
// wrappers, shared-memory matrix descriptors, and packed fp32 arithmetic.  Everything is
// written from the PTX ISA's descriptions of these instructions.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cstddef>
#include <cstdint>

#include "pad_internal.h"

namespace pad {
namespace tc {

constexpr unsigned long long kWaitNs = 1000000000ull;  // one second per bounded wait

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ unsigned long long globaltimer() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ float max3f(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// ---------------------------------------------------------------- packed fp32 pairs
// Blackwell executes two fp32 lanes per instruction (.f32x2); a pair lives in a b64.
__device__ __forceinline__ uint64_t f2pack(float lo, float hi) {
  return ((uint64_t)__float_as_uint(hi) << 32) | __float_as_uint(lo);
}
__device__ __forceinline__ float f2lo(uint64_t v) { return __uint_as_float((uint32_t)v); }
__device__ __forceinline__ float f2hi(uint64_t v) { return __uint_as_float((uint32_t)(v >> 32)); }
__device__ __forceinline__ uint64_t ffma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t fadd2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ uint64_t fadd2_rm(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rm.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}

// 2^x for a pair on the FMA pipe, to take part of the load off the MUFU unit.
// Cody-Waite split x = n + f with n = floor(x) and f in [0, 1): adding 1.5 * 2^23 with
// round-toward-minus-infinity leaves n in the low mantissa bits of t (exact for
// |x| < 2^22), and (bits(t) << 23) is n << 23 because the low nine bits of 1.5 * 2^23
// are zero.  2^f is a cubic fitted to 2^f on [0, 1) for the least maximum relative error
// (7.5e-5; 1.5e-4 after fp32 rounding), far below the bf16 rounding P gets next.
// x is clamped to -125: the cubic lies in [0.99, 2), so the exponent field stays normal.
constexpr float kExpC0 = 0.99992512554644490f;
constexpr float kExpC1 = 0.69583399210713630f;
constexpr float kExpC2 = 0.22606707273041300f;
constexpr float kExpC3 = 0.07802403102605904f;
__device__ __forceinline__ uint64_t exp2_poly2(uint64_t x) {
  const float x0 = fmaxf(f2lo(x), -125.f), x1 = fmaxf(f2hi(x), -125.f);
  const uint64_t xc = f2pack(x0, x1);
  const uint64_t magic = f2pack(12582912.f, 12582912.f);
  const uint64_t t = fadd2_rm(xc, magic);
  const uint64_t n = fadd2(t, f2pack(-12582912.f, -12582912.f));
  const uint64_t f = fadd2(xc, n ^ 0x8000000080000000ull);  // x - n
  uint64_t q = ffma2(f, f2pack(kExpC3, kExpC3), f2pack(kExpC2, kExpC2));
  q = ffma2(f, q, f2pack(kExpC1, kExpC1));
  q = ffma2(f, q, f2pack(kExpC0, kExpC0));
  const uint32_t lo = (uint32_t)q + ((uint32_t)t << 23);
  const uint32_t hi = (uint32_t)(q >> 32) + ((uint32_t)(t >> 32) << 23);
  return ((uint64_t)hi << 32) | lo;
}

// ---------------------------------------------------------------- mbarrier
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count));
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait for the phase of the given parity; false = gave up.  It gives up when the
// CTA's abort flag is raised, or after about one second, when it records
// PAD_ERR_DEVICE_TIMEOUT (tagged `where`) for the plan's generation and raises the flag
// itself, so that every other wait of the CTA gives up too.
static __device__ __noinline__ bool mbar_wait_slow(uint64_t* bar, uint32_t parity, int32_t* abort, uint64_t gen,
                                                   PadDevHeader* hdr, int where) {
  const unsigned long long t0 = globaltimer();
  for (uint32_t i = 1;; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 63u) == 0) {
      if (*reinterpret_cast<volatile int32_t*>(abort)) return false;
      if (globaltimer() - t0 > kWaitNs) {
        pad_set_error(hdr, gen, PAD_ERR_DEVICE_TIMEOUT, (int)blockIdx.x, where, (int)threadIdx.x);
        *reinterpret_cast<volatile int32_t*>(abort) = 1;
        return false;
      }
    }
  }
}
__device__ __forceinline__ bool mbar_wait_b(uint64_t* bar, uint32_t parity, int32_t* abort, uint64_t gen,
                                            PadDevHeader* hdr, int where) {
  if (mbar_try_wait(bar, parity)) return true;
  return mbar_wait_slow(bar, parity, abort, gen, hdr, where);
}
// Wait used while draining after an abort: bounded, reports nothing.
__device__ __forceinline__ void drain_wait(uint64_t* bar, uint32_t parity) {
  const unsigned long long t0 = globaltimer();
  while (!mbar_try_wait(bar, parity) && globaltimer() - t0 < kWaitNs) {
  }
}

// ---------------------------------------------------------------- TMA
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* map, int c0, int c1,
                                            int c2, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(smem_u32(bar))
      : "memory");
}

// ---------------------------------------------------------------- tcgen05
__device__ __forceinline__ void fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// Instruction descriptor of tcgen05.mma kind::f16: D fp32 (bits 4-5 = 1), A and B
// bf16 (bits 7-9, 10-12 = 1), K-major A (bit 15 = 0), B major-ness in bit 16,
// N >> 3 in bits 17-22, M >> 4 in bits 24-28.
constexpr uint32_t make_idesc(int M, int N, bool b_mn_major) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((b_mn_major ? 1u : 0u) << 16) |
         ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

// Shared-memory matrix descriptor: start address, leading / stride byte offsets,
// version 1 (bits 46-47), 128-byte swizzle (layout type 2 in bits 61-63).
__device__ __forceinline__ uint64_t sdesc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

__device__ __forceinline__ void mma_ss(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                       uint32_t idesc, uint32_t accum) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accum)
      : "memory");
}
__device__ __forceinline__ void mma_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc,
                                       uint32_t idesc, uint32_t accum) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}\n" ::"r"(d_tmem),
      "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accum)
      : "memory");
}
// The barrier completes once every MMA this thread issued before has completed.
__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t* r) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,"
      "%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
        "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
        "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t* r) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
      "%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]),
      "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]),
      "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]),
      "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t* r) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
      "%14,%15,%16};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]),
      "r"(r[15])
      : "memory");
}
// 16-lane shapes (a warp's 16 lanes from the address's lane, which stays in its quarter).
// 16x256b: thread t holds, for each repetition k (8 columns), lanes L + t/4 and L + 8 + t/4 at
// columns C + 8k + 2(t%4) and + 1, in the order (row, c), (row, c+1), (row+8, c), (row+8, c+1).
// 16x128b: per repetition k (4 columns), lanes L + t/4 and L + 8 + t/4 at column C + 4k + t%4.
__device__ __forceinline__ void tmem_ld16x256_x8(uint32_t taddr, uint32_t* r) {
  asm volatile(
      "tcgen05.ld.sync.aligned.16x256b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_st16x256_x8(uint32_t taddr, const uint32_t* r) {
  asm volatile(
      "tcgen05.st.sync.aligned.16x256b.x8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}
__device__ __forceinline__ void tmem_st16x128_x16(uint32_t taddr, const uint32_t* r) {
  asm volatile(
      "tcgen05.st.sync.aligned.16x128b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}
__device__ __forceinline__ void tmem_st16x128_x8(uint32_t taddr, const uint32_t* r) {
  asm volatile(
      "tcgen05.st.sync.aligned.16x128b.x8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
      : "memory");
}
__device__ __forceinline__ void tmem_wait_ld() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}
// The registers written by tcgen05.ld are valid only after tcgen05.wait::ld; listing them
// as operands of the wait makes every later use depend on it in the compiler's view too.
__device__ __forceinline__ void tmem_wait_ld_dep(uint32_t* r) {
  asm volatile(
      "tcgen05.wait::ld.sync.aligned;"
      : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]),
        "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]),
        "+r"(r[14]), "+r"(r[15]), "+r"(r[16]), "+r"(r[17]), "+r"(r[18]), "+r"(r[19]),
        "+r"(r[20]), "+r"(r[21]), "+r"(r[22]), "+r"(r[23]), "+r"(r[24]), "+r"(r[25]),
        "+r"(r[26]), "+r"(r[27]), "+r"(r[28]), "+r"(r[29]), "+r"(r[30]), "+r"(r[31])
      :
      : "memory");
}
__device__ __forceinline__ void tmem_wait_st() {
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// L2 prefetch of one line.
__device__ __forceinline__ void prefetch_l2(const void* a) {
  asm volatile("prefetch.global.L2 [%0];" ::"l"(a));
}

// Once its last K tile is issued (about three tiles before the CTA ends), the K producer
// warp asks L2 for what the branch/merge kernel after this grid will read first: for the
// (event, kv-head) task with the CTA's index, if there is one, the branch's stored K/V rows (through the page
// table, whose entries for those keys no kernel of this step writes), its Q rows and, in the
// one-call step, its new K/V row.  Those tasks then start on warm lines instead of waiting
// on HBM behind their page-table reads.  Page ids outside the pool are skipped.
__device__ __forceinline__ void prefetch_branch_tasks(const KParams& p, const __nv_bfloat16* q,
                                                   const __nv_bfloat16* kpool, const __nv_bfloat16* vpool,
                                                   int lane) {
  const int n_tasks = p.n_events * p.h_kv, G = p.group, ps = p.page_size;
  // one task per CTA at most: a warp that walked many tasks here would hold the CTA (and
  // the grid the branch/merge kernel waits for) open longer than the prefetch saves.  With
  // the fused tail, the task this CTA will run itself.
  const int t0 = p.fused ? plan_tasks(p)[blockIdx.x] : (int)blockIdx.x;
  for (int t = t0; t >= 0 && t < n_tasks && t < (int)gridDim.x; t += gridDim.x) {
    const int e = t / p.h_kv, h = t - (t / p.h_kv) * p.h_kv;
    const int len = plan_events(p)[e].len;
    const int32_t* ptab = p.page_table + (size_t)e * p.max_pages;
    for (int k = lane; k < len; k += 32) {
      const int pg = ptab[k / ps];
      if (pg < 0 || pg >= p.n_pages) continue;
      const size_t off = (((size_t)pg * p.h_kv + h) * ps + (k % ps)) * 128;
      prefetch_l2(kpool + off);
      prefetch_l2(kpool + off + 64);
      prefetch_l2(vpool + off);
      prefetch_l2(vpool + off + 64);
    }
    if (lane < 2 * G) prefetch_l2(q + ((size_t)e * p.h_q + h * G + (lane >> 1)) * 128 + 64 * (lane & 1));
    if (p.k_new != nullptr && lane < 4) {
      const __nv_bfloat16* src = static_cast<const __nv_bfloat16*>(lane < 2 ? p.k_new : p.v_new);
      prefetch_l2(src + ((size_t)e * p.h_kv + h) * 128 + 64 * (lane & 1));
    }
  }
}

}  // namespace tc

// Tensor maps of a token-major [tokens, h_kv, 128] bf16 K and V prefix (boxes of 64 head-dim
// columns x 1 head x 128 tokens, 128-byte swizzle), cached per (buffers, shape, device).
bool prefix_tensor_maps(const void* kp, const void* vp, int h_kv, int64_t tokens, int dev, CUtensorMap* mk,
                        CUtensorMap* mv);

}  // namespace pad
