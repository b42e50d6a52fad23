// a4 + a5 for one (event, kv-head), run by 256 threads (8 warps): used by the standalone
// branch/merge kernel (one CTA per task) and by the tensor-core prefix kernel, whose
// softmax warps take one task each after their prefix split.
//
//   a4, the own-branch part of the mask of Sec. 3.4: the branch's keys 0..len, its
//   private tokens and the one appended at this step (under the "causal attention" mask
//   of the ablation: the stored tokens of every branch of the video, then its own new
//   one), staged in rounds of kKeys (K and V rows through the page table, cp.async);
//   each warp takes 16 of a round's keys and
//   keeps a flash-attention state in registers in the manner of the warp-level MMA
//   kernels (the G <= 16 query rows form one m16 tile, S = Q K^T, online softmax on the
//   accumulators in base 2, O += P V with P re-packed from the S accumulators).
//   a5: the eight warp states and the prefix splits' partial states are merged by
//   log-sum-exp (Eq. for combining softmax states: M = max of the maxima, every state
//   weighted by 2^(m - M)), and O and the LSE are written once.
//
//   a2, when the step is one call (KParams::k_new set): key `len` is read from k_new /
//   v_new instead of the pools, and this task writes it into them (its page-table entry
//   too, by the kv-head-0 task of an event that took a new page).  No other task reads
//   this (event, kv-head)'s branch, so nothing else waits for that write.
//
// Staging before griddepcontrol.wait reads nothing the grids ahead write: Q rows, the
// branch's page ids (key `len`'s page is the one this step took, else the table's entry
// of an earlier step) and the K/V rows of keys 0..len-1, and key `len` itself when it
// comes from k_new / v_new.  In a one-call step that is all the branch pass reads, so the
// whole pass (and the merge of its warp states) runs before the wait.  After it: key `len`
// when the append kernel wrote it (two-call step, the branch pass follows), and the
// splits' (m, l) pairs and O rows once the caller says they are complete
// (`partials_ready`: at once for the standalone kernel, whose wait covers the prefix
// grid; after the split counters for the tensor-core kernel).
#pragma once

#include <cuda_bf16.h>
#include <cstddef>
#include <cstdint>

#include "pad_internal.h"

namespace pad {
namespace bm {

constexpr int kThreads = 256;                 // threads of one task (the default of 8 warps)
constexpr int kWarps = kThreads / 32;
constexpr int kKeys = 16 * kWarps;            // branch keys staged per round, at most
constexpr int kMaxChunk = 64;                 // prefix splits merged per staged chunk
constexpr float kNegInf = -__builtin_huge_valf();

__host__ __device__ constexpr size_t align16(size_t x) { return (x + 15) / 16 * 16; }
__host__ __device__ constexpr size_t max_sz(size_t a, size_t b) { return a > b ? a : b; }

// Shared memory of a task: this head, then three regions sized per launch (16-byte aligned):
//   kv   K rows [nkr][LD] and V rows [nkr][LD] of a round (nkr = KParams::branch_rows);
//        after the branch pass the warps' O rows, fp32 [warp][G][D]
//   ml   the splits' (m, l) pairs of a chunk, [G][sch]
//   po   the splits' O rows of a chunk, fp32 [sch][G][D]
template <int D>
struct Head {
  static constexpr int LD = D + 8;            // padded bf16 row: ldmatrix rows in distinct banks
  __nv_bfloat16 q[16][LD];
  int page[kKeys];
  int slot[kKeys];                            // offset of the key within its page
  float wm[kWarps][16], wl[kWarps][16];       // each warp's branch state per row
  float sc[16][kMaxChunk];                    // state weights 2^(m - M)
  alignas(16) float ob[16][D];                // merged numerator (read as float4)
  float M[16], L[16], a[16];
};
// Keys staged per round by a task of NW warps (16 per warp), for a launch's branch_rows.
__host__ __device__ constexpr int round_keys(int branch_rows, int NW) {
  return branch_rows < 16 * NW ? branch_rows : 16 * NW;
}
template <int D, int NW = kWarps>
__host__ __device__ constexpr size_t kv_bytes(int nkr, int G) {
  return align16(max_sz((size_t)2 * nkr * Head<D>::LD * 2, (size_t)NW * G * D * 4));
}
template <int D, int NW = kWarps>
__host__ __device__ constexpr size_t smem_bytes(int branch_rows, int G, int sch) {
  return align16(sizeof(Head<D>)) + kv_bytes<D, NW>(round_keys(branch_rows, NW), G) + align16((size_t)G * sch * 8) +
         (size_t)sch * G * D * 4;
}

#ifdef __CUDACC__
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ void cp_async16(void* smem, const void* gmem, bool pred) {
  unsigned s = static_cast<unsigned>(__cvta_generic_to_shared(smem));
  int n = pred ? 16 : 0;
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(s), "l"(gmem), "r"(n));
}
__device__ __forceinline__ void cp_async8(void* smem, const void* gmem) {
  unsigned s = static_cast<unsigned>(__cvta_generic_to_shared(smem));
  asm volatile("cp.async.ca.shared.global [%0], [%1], 8;\n" ::"r"(s), "l"(gmem));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;\n" ::"n"(N));
}
__device__ __forceinline__ void ldsm_x4(uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3,
                                        const void* p) {
  unsigned a = static_cast<unsigned>(__cvta_generic_to_shared(p));
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(a));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3,
                                          const void* p) {
  unsigned a = static_cast<unsigned>(__cvta_generic_to_shared(p));
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(a));
}
__device__ __forceinline__ void mma_bf16(float* c, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
// Partial row of part `split` of (video, kv-head), row r.
__device__ __forceinline__ int64_t part_row(const PadVideoDesc& vd, int kvh, int split, int R, int r) {
  return (int64_t)vd.part_base + ((int64_t)kvh * vd.n_splits + split) * R + r;
}

// Barriers over the task's 256 threads: the whole CTA, or a named barrier.
struct SyncCta {
  __device__ void sync() const { __syncthreads(); }
  __device__ bool all(bool v) const { return __syncthreads_and(v) != 0; }
};
struct SyncNamed {
  int id;
  __device__ void sync() const { asm volatile("bar.sync %0, 256;" ::"r"(id) : "memory"); }
  __device__ bool all(bool v) const {
    int r;
    asm volatile(
        "{\n .reg .pred pi, po;\n setp.ne.s32 pi, %1, 0;\n bar.red.and.pred po, %2, 256, pi;\n"
        " selp.s32 %0, 1, 0, po;\n}\n"
        : "=r"(r)
        : "r"((int)v), "r"(id)
        : "memory");
    return r != 0;
  }
};

// One task.  `tid` in [0, 256); `smem` 16-byte aligned, smem_bytes<D>(branch_rows, G, sch)
// long.  `partials_ready()` is called by all 256 threads and returns false if the
// partials cannot be read (then only the status word is written).
// CAUSAL: 0 = the method's own-branch keys, 1 = the causal-attention key list, 2 = read
// KParams::causal at run time (separate instantiations keep the common one lean).
template <int D, bool ROPE, int CAUSAL, int NW = kWarps, class Sync, class Ready>
__device__ __forceinline__ void run_task(const KParams& p, const __nv_bfloat16* __restrict__ q,
                                         const __nv_bfloat16* __restrict__ kpool,
                                         const __nv_bfloat16* __restrict__ vpool, void* __restrict__ out,
                                         float* __restrict__ lse, int e, int kvh, int tid,
                                         unsigned char* smem, int sch, const Sync& sy, bool early,
                                         Ready partials_ready) {
  static_assert(NW >= 1 && NW <= kWarps, "warps per task");
  constexpr int NT = 32 * NW;
  constexpr int CH = D / 8;                   // 16-byte pieces of a bf16 row
  constexpr int KS = D / 16;                  // k-steps of S = Q K^T
  constexpr int OT = D / 8;                   // n8 tiles of O
  constexpr int D4 = D / 4;
  constexpr int LD = Head<D>::LD;
  Head<D>& S = *reinterpret_cast<Head<D>*>(smem);
  const int G = p.group;
  const int nkr = round_keys(p.branch_rows, NW);  // keys per round (multiple of 16, <= 16 NW)
  unsigned char* kv_raw = smem + align16(sizeof(Head<D>));
  __nv_bfloat16 (*sK)[LD] = reinterpret_cast<__nv_bfloat16 (*)[LD]>(kv_raw);
  __nv_bfloat16 (*sV)[LD] = reinterpret_cast<__nv_bfloat16 (*)[LD]>(kv_raw + (size_t)nkr * LD * 2);
  float* wo = reinterpret_cast<float*>(kv_raw);  // [warp][G][d] after the branch pass
  float2* sml = reinterpret_cast<float2*>(kv_raw + kv_bytes<D, NW>(nkr, G));
  float* spo = reinterpret_cast<float*>(reinterpret_cast<unsigned char*>(sml) + align16((size_t)G * sch * 8));

  const int warp = tid >> 5, lane = tid & 31;
  const int gq = lane >> 2, t4 = lane & 3;
  const PadEventDesc ev = plan_events(p)[e];
  const PadVideoDesc vd = plan_videos(p)[ev.video];
  const int R = vd.n_events * G;
  const int ns = vd.n_splits;
  const int rbase = ev.local * G;
  const int len = ev.len;                     // keys before this step; key `len` is this step's
  const int ps = p.page_size;
  // The task's keys: its own branch's len + 1, or (causal mask) the stored tokens of every
  // branch of the video, branch by branch, then its own token of this step.  `own` is the
  // index of that token among them.
  const bool causal = CAUSAL == 2 ? p.causal != 0 : CAUSAL == 1;
  int own = len;
  if (causal) {
    own = 0;
    for (int f = 0; f < vd.n_events; ++f) own += plan_events(p)[vd.first_event + f].len;
  }
  const int nk = own + 1;

  // page of task key `key` (-1 if out of the pool) and, in `slot`, its offset in the page
  auto page_of = [&](int key, int& slot) -> int {
    int row = e, t = key;
    if (causal) {
      if (key == own) {
        t = len;
      } else {
        row = vd.first_event;
        for (int lf = plan_events(p)[row].len; t >= lf; lf = plan_events(p)[row].len) {
          t -= lf;
          ++row;
        }
      }
    }
    slot = t % ps;
    const int pi = t / ps;
    int page = (row == e && pi == len / ps && ev.new_page >= 0) ? ev.new_page
                                                              : p.page_table[(size_t)row * p.max_pages + pi];
    if (page < 0 || page >= p.n_pages) {
      pad_set_error(p.header, p.gen, PAD_ERR_DEVICE_BOUNDS, row, pi, page);
      page = -1;
    }
    return page;
  };
  auto locate = [&](int r0, int nv) {         // page ids and offsets of a round's keys
    if (tid < nkr) {
      int sl = 0;
      S.page[tid] = tid < nv ? page_of(r0 + tid, sl) : -1;
      S.slot[tid] = sl;
    }
  };
  const int nv0 = min(nkr, nk);
  locate(0, nv0);
  // (ROPE: the plan carries positions; a separate instantiation keeps the plain one lean)
  const float* cs = ROPE ? p.rope_cs + (size_t)ev.pos * D : nullptr;
  for (int i = tid; i < 16 * CH; i += NT) {
    const int g = i / CH, c = i - (i / CH) * CH;
    const bool in = g < G;
    const __nv_bfloat16* qr = q + ((size_t)e * p.h_q + kvh * G + (in ? g : 0)) * D;
    if (ROPE)  // rotated here (rows past G are zero)
      *reinterpret_cast<uint4*>(&S.q[g][c * 8]) = in ? rope_chunk8(qr, D, c * 8, cs) : make_uint4(0u, 0u, 0u, 0u);
    else
      cp_async16(&S.q[g][c * 8], qr + c * 8, in);
  }
  for (int i = tid; i < G * D; i += NT) S.ob[i / D][i % D] = 0.f;
  if (tid < 16) {
    S.M[tid] = kNegInf;
    S.L[tid] = 0.f;
  }
  sy.sync();
  const __nv_bfloat16* knew = static_cast<const __nv_bfloat16*>(p.k_new);
  const __nv_bfloat16* vnew = static_cast<const __nv_bfloat16*>(p.v_new);
  const size_t new_row = ((size_t)e * p.h_kv + kvh) * D;
  auto stage_keys = [&](int r0, int nv, int k_lo, int k_hi) {  // rows k_lo..k_hi-1 of the round
    for (int i = tid; i < (k_hi - k_lo) * CH; i += NT) {
      const int k = k_lo + i / CH, c = i - (i / CH) * CH;
      const int pg = k < nv ? S.page[k] : -1;
      const bool in = pg >= 0;
      if (knew != nullptr && r0 + k == own) {
        if (ROPE)
          *reinterpret_cast<uint4*>(&sK[k][c * 8]) = in ? rope_chunk8(knew + new_row, D, c * 8, cs)
                                                        : make_uint4(0u, 0u, 0u, 0u);
        else
          cp_async16(&sK[k][c * 8], knew + new_row + c * 8, in);
        cp_async16(&sV[k][c * 8], vnew + new_row + c * 8, in);
        continue;
      }
      const size_t off = (((size_t)(in ? pg : 0) * p.h_kv + kvh) * ps + (in ? S.slot[k] : 0)) * D + c * 8;
      cp_async16(&sK[k][c * 8], kpool + off, in);
      cp_async16(&sV[k][c * 8], vpool + off, in);
    }
  };
  if (knew != nullptr) {
    // a2: this task's row of the new token into the pools (16-byte pieces of K, then V);
    // its page was located with the first round's keys when it is among them
    if (tid < 2 * CH) {
      int sl = 0;
      const int pg = own < nkr ? S.page[own] : page_of(own, sl);
      if (pg >= 0) {
        const int c = tid % CH;
        const bool isv = tid >= CH;
        const size_t dst = (((size_t)pg * p.h_kv + kvh) * ps + (len % ps)) * D + c * 8;
        const uint4 v = (ROPE && !isv) ? rope_chunk8(knew + new_row, D, c * 8, cs)
                                                : *reinterpret_cast<const uint4*>((isv ? vnew : knew) + new_row + c * 8);
        *reinterpret_cast<uint4*>(const_cast<__nv_bfloat16*>(isv ? vpool : kpool) + dst) = v;
      }
    }
    if (kvh == 0 && tid == 0 && ev.new_page >= 0 && ev.new_page < p.n_pages)
      p.page_table[(size_t)e * p.max_pages + len / ps] = ev.new_page;
  }
  const int nv0_16 = (nv0 + 15) & ~15;
  // this step's key waits for the grids ahead only when the append kernel wrote it
  const bool len_in_first = own < nkr && knew == nullptr;
  // rows 0..nv0_16-1 except that key (rows past nv0 are zero-filled)
  if (len_in_first) {
    stage_keys(0, nv0, 0, own);
    stage_keys(0, nv0, own + 1, nv0_16);
  } else {
    stage_keys(0, nv0, 0, nv0_16);
  }
  cp_async_commit();
  // One-call step: nothing the branch pass reads is written by the grids ahead, so the
  // whole pass runs before the wait and only the merge of the splits' partials follows it;
  // unless the plan says this CTA cannot start before the prefix grid completes anyway
  // (merge_first), where waiting first lets the partials load during the branch pass.
  const bool pre = knew != nullptr && !p.merge_first;

  // ---------------- after the grids ahead (at least the append) completed
  if (!pre) {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    if (len_in_first) stage_keys(0, nv0, own, own + 1);
  }
  cp_async_commit();                          // this round's keys

  // the splits' O rows and (m, l) pairs of chunk [s0, s0 + nch): per split, the task's G
  // rows are one contiguous block of G * D floats, R * D floats after the previous split's
  // (the flat index is advanced by NT without a division)
  auto stage_chunk = [&](int s0, int nch) {
    const int gd4 = G * D4;
    const float* base = p.part_o + part_row(vd, kvh, s0, R, rbase) * D;
    const size_t split_stride = (size_t)R * D;
    int sl = tid / gd4, r = tid - (tid / gd4) * gd4;
    const int adv_sl = NT / gd4, adv_r = NT - (NT / gd4) * gd4;
    for (; sl < nch;) {
      cp_async16(spo + (size_t)sl * G * D + (size_t)r * 4, base + sl * split_stride + (size_t)r * 4, true);
      sl += adv_sl;
      r += adv_r;
      if (r >= gd4) {
        r -= gd4;
        ++sl;
      }
    }
    const float2* mbase = p.part_ml + part_row(vd, kvh, s0, R, rbase);
    for (int i = tid; i < G * nch; i += NT) {
      const int g = i / nch, k = i - g * nch;
      cp_async8(&sml[g * sch + k], mbase + (size_t)k * R + g);
    }
  };
  bool ok = true;
  if (early && !pre) {
    if (ns > 0) stage_chunk(0, min(sch, ns));
    cp_async_commit();                        // the first chunk, waited for in a5
  }

  // ---------------- a4: the branch pass
  float o[OT][4];
#pragma unroll
  for (int i = 0; i < OT; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float m_lo = kNegInf, m_hi = kNegInf;       // rows gq, gq + 8 (log2 units)
  float l_lo = 0.f, l_hi = 0.f;               // this lane's share of the row sums
  uint32_t qa[KS][4];
  const int kb0 = 16 * warp;                  // this warp's keys within a round
  for (int r0 = 0; r0 < nk; r0 += nkr) {
    const int nv = min(nkr, nk - r0);
    if (r0 > 0) {
      locate(r0, nv);
      sy.sync();
      stage_keys(r0, nv, 0, (nv + 15) & ~15);
      cp_async_commit();
      cp_async_wait<0>();
    } else if (early && !pre) {
      cp_async_wait<1>();                     // all but the first chunk's group
    } else {
      cp_async_wait<0>();
    }
    sy.sync();
    if (r0 == 0) {
#pragma unroll
      for (int kk = 0; kk < KS; ++kk)
        ldsm_x4(qa[kk][0], qa[kk][1], qa[kk][2], qa[kk][3], &S.q[lane & 15][kk * 16 + (lane >> 4) * 8]);
    }
    if (kb0 < nv) {
      float s[2][4];
#pragma unroll
      for (int nt = 0; nt < 2; ++nt) {
        s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
#pragma unroll
        for (int kk = 0; kk < KS; kk += 2) {
          uint32_t b0, b1, b2, b3;
          ldsm_x4(b0, b1, b2, b3, &sK[kb0 + nt * 8 + (lane & 7)][kk * 16 + (lane >> 3) * 8]);
          mma_bf16(s[nt], qa[kk], b0, b1);
          mma_bf16(s[nt], qa[kk + 1], b2, b3);
        }
      }
      float mx_lo = kNegInf, mx_hi = kNegInf;
#pragma unroll
      for (int nt = 0; nt < 2; ++nt) {
#pragma unroll
        for (int j = 0; j < 2; ++j) {
          const int k = kb0 + nt * 8 + 2 * t4 + j;
          const bool in = k < nv && S.page[k] >= 0;
          s[nt][j] = in ? s[nt][j] * p.scale_log2 : kNegInf;
          s[nt][2 + j] = in ? s[nt][2 + j] * p.scale_log2 : kNegInf;
          mx_lo = fmaxf(mx_lo, s[nt][j]);
          mx_hi = fmaxf(mx_hi, s[nt][2 + j]);
        }
      }
      mx_lo = fmaxf(mx_lo, __shfl_xor_sync(0xffffffffu, mx_lo, 1));
      mx_lo = fmaxf(mx_lo, __shfl_xor_sync(0xffffffffu, mx_lo, 2));
      mx_hi = fmaxf(mx_hi, __shfl_xor_sync(0xffffffffu, mx_hi, 1));
      mx_hi = fmaxf(mx_hi, __shfl_xor_sync(0xffffffffu, mx_hi, 2));
      float mn_lo = fmaxf(m_lo, mx_lo), mn_hi = fmaxf(m_hi, mx_hi);
      if (mn_lo == kNegInf) mn_lo = 0.f;  // only while every key so far failed its bounds check
      if (mn_hi == kNegInf) mn_hi = 0.f;
      const float al_lo = ex2(m_lo - mn_lo), al_hi = ex2(m_hi - mn_hi);
      m_lo = mn_lo;
      m_hi = mn_hi;
      float pr[2][4];
#pragma unroll
      for (int h = 0; h < 2; ++h)
#pragma unroll
        for (int j = 0; j < 4; ++j) pr[h][j] = ex2(s[h][j] - (j < 2 ? mn_lo : mn_hi));
      l_lo = l_lo * al_lo + (pr[0][0] + pr[0][1]) + (pr[1][0] + pr[1][1]);
      l_hi = l_hi * al_hi + (pr[0][2] + pr[0][3]) + (pr[1][2] + pr[1][3]);
      uint32_t a[4];
      a[0] = pack_bf16(pr[0][0], pr[0][1]);
      a[1] = pack_bf16(pr[0][2], pr[0][3]);
      a[2] = pack_bf16(pr[1][0], pr[1][1]);
      a[3] = pack_bf16(pr[1][2], pr[1][3]);
#pragma unroll
      for (int i = 0; i < OT; i += 2) {
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(b0, b1, b2, b3, &sV[kb0 + (lane & 15)][(i + (lane >> 4)) * 8]);
        o[i][0] *= al_lo;
        o[i][1] *= al_lo;
        o[i][2] *= al_hi;
        o[i][3] *= al_hi;
        o[i + 1][0] *= al_lo;
        o[i + 1][1] *= al_lo;
        o[i + 1][2] *= al_hi;
        o[i + 1][3] *= al_hi;
        mma_bf16(o[i], a, b0, b1);
        mma_bf16(o[i + 1], a, b2, b3);
      }
    }
    sy.sync();                                // the next round (or the O rows below) overwrite k / v
  }
  l_lo += __shfl_xor_sync(0xffffffffu, l_lo, 1);
  l_lo += __shfl_xor_sync(0xffffffffu, l_lo, 2);
  l_hi += __shfl_xor_sync(0xffffffffu, l_hi, 1);
  l_hi += __shfl_xor_sync(0xffffffffu, l_hi, 2);
  // this warp's state: (m, l) per row and its O rows
  if (t4 == 0) {
    S.wm[warp][gq] = m_lo;
    S.wl[warp][gq] = l_lo;
    S.wm[warp][gq + 8] = m_hi;
    S.wl[warp][gq + 8] = l_hi;
  }
  if (gq < G) {
    float* dst = wo + ((size_t)warp * G + gq) * D;
#pragma unroll
    for (int i = 0; i < OT; ++i) *reinterpret_cast<float2*>(dst + i * 8 + 2 * t4) = make_float2(o[i][0], o[i][1]);
  }
  if (gq + 8 < G) {
    float* dst = wo + ((size_t)warp * G + gq + 8) * D;
#pragma unroll
    for (int i = 0; i < OT; ++i) *reinterpret_cast<float2*>(dst + i * 8 + 2 * t4) = make_float2(o[i][2], o[i][3]);
  }
  sy.sync();

  // ---------------- a5: the warp states, then the prefix splits in chunks of `sch`
  for (int g = warp; g < G; g += NW) {
    const float mw = lane < NW ? S.wm[lane][g] : kNegInf;
    float mx = warp_max(mw);
    if (mx == kNegInf) mx = 0.f;              // no key of the branch passed its bounds check
    const float wgt = lane < NW ? ex2(mw - mx) : 0.f;
    const float sum = warp_sum(lane < NW ? S.wl[lane][g] * wgt : 0.f);
    if (lane < NW) S.sc[g][lane] = wgt;
    if (lane == 0) {
      S.M[g] = mx;
      S.L[g] = sum;
    }
  }
  sy.sync();
  for (int i = tid; i < G * D4; i += NT) {
    const int g = i / D4, d4 = i - g * D4;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int w = 0; w < NW; ++w) {
      const float c = S.sc[g][w];
      const float4 v = reinterpret_cast<const float4*>(wo)[(w * G + g) * D4 + d4];
      acc.x = fmaf(c, v.x, acc.x);
      acc.y = fmaf(c, v.y, acc.y);
      acc.z = fmaf(c, v.z, acc.z);
      acc.w = fmaf(c, v.w, acc.w);
    }
    reinterpret_cast<float4*>(&S.ob[g][0])[d4] = acc;
  }

  if (early && pre) {
    // ---------------- after the grids ahead (the prefix pass) completed
    asm volatile("griddepcontrol.wait;" ::: "memory");
    if (ns > 0) stage_chunk(0, min(sch, ns));
    cp_async_commit();
  }
  if (!early && ns > 0) {
    ok = partials_ready();
    if (ok) stage_chunk(0, min(sch, ns));
    cp_async_commit();
  }
  for (int s0 = 0; ok && s0 < ns; s0 += sch) {
    const int nch = min(sch, ns - s0);
    if (s0 > 0) {
      sy.sync();                              // the previous chunk's rows are consumed
      stage_chunk(s0, nch);
    }
    cp_async_commit();
    cp_async_wait<0>();
    sy.sync();
    // row statistics, one warp per row, lanes over splits
    for (int g = warp; g < G; g += NW) {
      float mx = kNegInf;
      for (int sl = lane; sl < nch; sl += 32) mx = fmaxf(mx, sml[g * sch + sl].x);
      mx = warp_max(mx);
      const float mo = S.M[g];
      const float mn = fmaxf(mo, mx);
      float sum = 0.f;
      for (int sl = lane; sl < nch; sl += 32) {
        const float2 ml = sml[g * sch + sl];
        const float wgt = ex2(ml.x - mn);
        S.sc[g][sl] = wgt;
        sum = fmaf(ml.y, wgt, sum);
      }
      sum = warp_sum(sum);
      if (lane == 0) {
        const float al = ex2(mo - mn);
        S.a[g] = al;
        S.L[g] = S.L[g] * al + sum;
        S.M[g] = mn;
      }
    }
    sy.sync();
    for (int i = tid; i < G * D4; i += NT) {
      const int g = i / D4, d4 = i - g * D4;
      const float4* src = reinterpret_cast<const float4*>(spo) + g * D4 + d4;
      const int step = G * D4;
      const float al = S.a[g];
      float4 acc = reinterpret_cast<const float4*>(&S.ob[g][0])[d4];
      acc.x *= al;
      acc.y *= al;
      acc.z *= al;
      acc.w *= al;
#pragma unroll 4
      for (int sl = 0; sl < nch; ++sl) {
        const float c = S.sc[g][sl];
        const float4 v = src[sl * step];
        acc.x = fmaf(c, v.x, acc.x);
        acc.y = fmaf(c, v.y, acc.y);
        acc.z = fmaf(c, v.z, acc.z);
        acc.w = fmaf(c, v.w, acc.w);
      }
      reinterpret_cast<float4*>(&S.ob[g][0])[d4] = acc;
    }
  }
  cp_async_wait<0>();
  sy.sync();
  if (!ok) return;

  for (int i = tid; i < G * D4; i += NT) {
    const int g = i / D4, d4 = i - g * D4;
    const float inv = 1.0f / S.L[g];
    float4 v = reinterpret_cast<const float4*>(&S.ob[g][0])[d4];
    v.x *= inv;
    v.y *= inv;
    v.z *= inv;
    v.w *= inv;
    const size_t oi = ((size_t)e * p.h_q + kvh * G + g) * D + 4 * d4;
    if (p.out_bf16)
      *reinterpret_cast<uint2*>(reinterpret_cast<__nv_bfloat16*>(out) + oi) =
          make_uint2(pack_bf16(v.x, v.y), pack_bf16(v.z, v.w));
    else
      *reinterpret_cast<float4*>(reinterpret_cast<float*>(out) + oi) = v;
    if (lse != nullptr && d4 == 0)
      lse[(size_t)e * p.h_q + kvh * G + g] = (S.M[g] + log2f(S.L[g])) * 0.69314718055994531f;
  }
}
#endif  // __CUDACC__

}  // namespace bm
}  // namespace pad
