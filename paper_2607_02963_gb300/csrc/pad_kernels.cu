// Kernels of one event-factorized decode step (Sec. 3.4, Eq. 3):
//   host_in_kernel       the step inputs from device-mapped host memory (pad_step_run_host)
//   append_kernel        a2: scatter each branch's new K/V into its page, write new page-table entries
//   prefix_simt_kernel   a3 for few rows (R = E_b * G <= 16): warp-shuffle split-KV flash-decode
//   prefix_mma_kernel    a3 with warp-level mma.sync (m16n8k16, bf16 in, fp32 accumulate)
//   branch_merge_kernel  a4 + a5: each branch's private-suffix pass, then the log-sum-exp merge
//                        of its prefix partials (the mask of Fig. 3: own branch only)
//
// Partial softmax states (m, l, O) keep m in log2 units of the scaled score:
// m = max_k s_k * scale * log2(e), l = sum_k 2^(s_k*scale*log2(e) - m), O = sum_k 2^(...) v_k.
#include <cuda_bf16.h>
#include <cstddef>
#include <cstdint>

#include <algorithm>

#include "pad_branch_merge.cuh"
#include "pad_internal.h"

namespace pad {

namespace {

constexpr float kNegInf = -__builtin_huge_valf();


// Hardware base-2 exponential (MUFU.EX2); exp2(-inf) = 0.
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

__device__ __forceinline__ void unpack8(const uint4& r, float* f) {
  f[0] = bf16_lo(r.x); f[1] = bf16_hi(r.x);
  f[2] = bf16_lo(r.y); f[3] = bf16_hi(r.y);
  f[4] = bf16_lo(r.z); f[5] = bf16_hi(r.z);
  f[6] = bf16_lo(r.w); f[7] = bf16_hi(r.w);
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

// Query row r of (video, kv-head): event e_local = r / G, head kvh*G + r % G.
__device__ __forceinline__ const __nv_bfloat16* q_row(const KParams& p, int first_event,
                                                      const __nv_bfloat16* q, int kvh, int r) {
  int el = r / p.group;
  int gh = r - el * p.group;
  return q + ((size_t)(first_event + el) * p.h_q + kvh * p.group + gh) * p.head_dim;
}

__device__ __forceinline__ int64_t part_row(const PadVideoDesc& vd, int kvh, int split, int R, int r) {
  return (int64_t)vd.part_base + ((int64_t)kvh * vd.n_splits + split) * R + r;
}

// ---------------------------------------------------------------------------
// a2: fused append.  One thread per 16-byte chunk of one (event, kv-head) row.
// ---------------------------------------------------------------------------
__global__ void append_kernel(const __grid_constant__ KParams p, const uint4* __restrict__ k_new,
                              const uint4* __restrict__ v_new, uint4* __restrict__ k_pool,
                              uint4* __restrict__ v_pool) {
  // the shared-prefix pass launched after this kernel reads nothing it writes before its
  // griddepcontrol.wait
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int chunks = p.head_dim / 8;
  const int per_event = p.h_kv * chunks;
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  // the split counters of the fused tail start the step at zero (there are fewer of them
  // than threads here: at most h_kv per event)
  if (idx < p.n_counters) p.counters[idx] = 0u;
  if (idx >= p.n_events * per_event) return;
  const int e = idx / per_event;
  const int rem = idx - e * per_event;
  const int h = rem / chunks;
  const int c = rem - h * chunks;
  const PadEventDesc ev = plan_events(p)[e];
  const int pidx = ev.len / p.page_size;
  const int slot = ev.len - pidx * p.page_size;
  int page;
  if (ev.new_page >= 0) {
    page = ev.new_page;
    if (rem == 0) p.page_table[(size_t)e * p.max_pages + pidx] = page;
  } else {
    page = p.page_table[(size_t)e * p.max_pages + pidx];
  }
  if (page < 0 || page >= p.n_pages) {
    pad_set_error(p.header, p.gen, PAD_ERR_DEVICE_BOUNDS, e, pidx, page);
    return;
  }
  const size_t dst = (((size_t)page * p.h_kv + h) * p.page_size + slot) * chunks + c;
  const size_t src = ((size_t)e * p.h_kv + h) * chunks + c;
  k_pool[dst] = p.rope_cs != nullptr
                    ? rope_chunk8(reinterpret_cast<const __nv_bfloat16*>(k_new + (src - c)), p.head_dim, 8 * c,
                                  p.rope_cs + (size_t)ev.pos * p.head_dim)
                    : k_new[src];
  v_pool[dst] = v_new[src];
}

// ---------------------------------------------------------------------------
// a3, few rows: warp-shuffle split-KV flash-decode.  One CTA (8 warps) per work
// item; warp w takes 32-token chunks w, w+8, ...; lane = token for q.k, lane =
// head_dim slice for p.v; the 8 warps' states are merged through shared memory.
// ---------------------------------------------------------------------------
template <int D, int MAXR>
__global__ void __launch_bounds__(256) prefix_simt_kernel(const __grid_constant__ KParams p,
                                                          const __nv_bfloat16* __restrict__ q,
                                                          const __nv_bfloat16* __restrict__ kp,
                                                          const __nv_bfloat16* __restrict__ vp) {
  constexpr int NW = 8;
  constexpr int VPL = D / 32;  // head_dim elements per lane in p.v
  __shared__ float sq[MAXR][D];
  __shared__ float sp[NW][MAXR][32];
  __shared__ float sm[NW][MAXR];
  __shared__ float sl[NW][MAXR];
  __shared__ float so[MAXR][D];
  __shared__ GMask sg[MAXR];

  const PadWorkItem it = plan_items(p)[blockIdx.x];
  const int R = it.n_events * p.group;
  const int kvh = it.kvh;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x < MAXR) {
    GMask g{0, 0, -1};
    if (p.g_self && (int)threadIdx.x < R) {
      const PadEventDesc ev = plan_events(p)[it.first_event + threadIdx.x / p.group];
      g = g_mask_of(p, plan_videos(p)[ev.video], ev);
    }
    sg[threadIdx.x] = g;
  }

  for (int i = threadIdx.x; i < MAXR * D; i += blockDim.x) {
    int r = i / D, d = i - r * D;
    float v = 0.f;
    if (r < R) {
      const __nv_bfloat16* qr = q_row(p, it.first_event, q, kvh, r);
      v = p.rope_cs != nullptr
              ? rope_elem(qr, D, d, p.rope_cs + (size_t)plan_events(p)[it.first_event + r / p.group].pos * D)
              : __bfloat162float(qr[d]);
    }
    sq[r][d] = v;
    so[r][d] = 0.f;
  }
  __syncthreads();

  float o[MAXR][VPL];
  float m[MAXR], l[MAXR];
#pragma unroll
  for (int r = 0; r < MAXR; ++r) {
    m[r] = kNegInf;
    l[r] = 0.f;
#pragma unroll
    for (int i = 0; i < VPL; ++i) o[r][i] = 0.f;
  }

  const int ntok = it.tok_end - it.tok_begin;
  const size_t row_stride = (size_t)p.h_kv * D;
  const __nv_bfloat16* kbase = kp + (size_t)it.tok0 * row_stride + (size_t)kvh * D;
  const __nv_bfloat16* vbase = vp + (size_t)it.tok0 * row_stride + (size_t)kvh * D;

  for (int c0 = warp * 32; c0 < ntok; c0 += NW * 32) {
    const int t = c0 + lane;
    const bool valid = t < ntok;
    float s[MAXR];
#pragma unroll
    for (int r = 0; r < MAXR; ++r) s[r] = 0.f;
    if (valid) {
      const uint4* kr = reinterpret_cast<const uint4*>(kbase + (size_t)t * row_stride);
#pragma unroll 4
      for (int d8 = 0; d8 < D / 8; ++d8) {
        float kf[8];
        unpack8(__ldg(kr + d8), kf);
#pragma unroll
        for (int r = 0; r < MAXR; ++r) {
          if (r < R) {
#pragma unroll
            for (int j = 0; j < 8; ++j) s[r] = fmaf(sq[r][d8 * 8 + j], kf[j], s[r]);
          }
        }
      }
    }
#pragma unroll
    for (int r = 0; r < MAXR; ++r) {
      if (r < R) {
        float sv = valid && g_visible(sg[r], it.tok_begin + t) ? s[r] * p.scale_log2 : kNegInf;
        float mn = fmaxf(m[r], warp_max(sv));
        // -inf only while every token so far was hidden by the self G-token mask
        const float mb = mn == kNegInf ? 0.f : mn;
        float alpha = ex2(m[r] - mb);
        float pr = ex2(sv - mb);
        l[r] = l[r] * alpha + warp_sum(pr);
        m[r] = mn;
#pragma unroll
        for (int i = 0; i < VPL; ++i) o[r][i] *= alpha;
        sp[warp][r][lane] = pr;
      }
    }
    __syncwarp();
    const int nv = min(32, ntok - c0);
    for (int j = 0; j < nv; ++j) {
      const __nv_bfloat16* vr = vbase + (size_t)(c0 + j) * row_stride + lane * VPL;
      float vf[VPL];
      if constexpr (VPL == 4) {
        uint2 raw = __ldg(reinterpret_cast<const uint2*>(vr));
        vf[0] = bf16_lo(raw.x); vf[1] = bf16_hi(raw.x); vf[2] = bf16_lo(raw.y); vf[3] = bf16_hi(raw.y);
      } else {
        uint32_t raw = __ldg(reinterpret_cast<const unsigned int*>(vr));
        vf[0] = bf16_lo(raw); vf[1] = bf16_hi(raw);
      }
#pragma unroll
      for (int r = 0; r < MAXR; ++r) {
        if (r < R) {
          float pj = sp[warp][r][j];
#pragma unroll
          for (int i = 0; i < VPL; ++i) o[r][i] = fmaf(pj, vf[i], o[r][i]);
        }
      }
    }
    __syncwarp();
  }

  if (lane == 0) {
#pragma unroll
    for (int r = 0; r < MAXR; ++r) {
      sm[warp][r] = m[r];
      sl[warp][r] = l[r];
    }
  }
  __syncthreads();
  // deterministic combination of the warps' states (fixed order: warp 0, 1, ...)
  for (int w = 0; w < NW; ++w) {
    if (warp == w) {
#pragma unroll
      for (int r = 0; r < MAXR; ++r) {
        if (r < R) {
          float M = kNegInf;
#pragma unroll
          for (int u = 0; u < NW; ++u) M = fmaxf(M, sm[u][r]);
          const float f = (m[r] == kNegInf) ? 0.f : ex2(m[r] - M);
#pragma unroll
          for (int i = 0; i < VPL; ++i) so[r][lane * VPL + i] += o[r][i] * f;
        }
      }
    }
    __syncthreads();
  }
  for (int i = threadIdx.x; i < R * D; i += blockDim.x) {
    int r = i / D, d = i - r * D;
    float M = kNegInf;
#pragma unroll
    for (int w = 0; w < NW; ++w) M = fmaxf(M, sm[w][r]);
    int64_t pr = (int64_t)it.part_row0 + r;
    if (d == 0) {
      float L = 0.f;
#pragma unroll
      for (int w = 0; w < NW; ++w)
        if (sm[w][r] != kNegInf) L += sl[w][r] * ex2(sm[w][r] - M);
      p.part_ml[pr] = make_float2(M, L);
    }
    p.part_o[pr * D + d] = so[r][d];
  }
}

// ---------------------------------------------------------------------------
// a3, tensor path on the warp-level MMA: one CTA per (work item, 64-row block);
// 4 warps x 16 query rows; 64-token K/V tiles double-buffered with cp.async.
// ---------------------------------------------------------------------------
template <int D>
__global__ void __launch_bounds__(128) prefix_mma_kernel(const __grid_constant__ KParams p,
                                                         const __nv_bfloat16* __restrict__ q,
                                                         const __nv_bfloat16* __restrict__ kp,
                                                         const __nv_bfloat16* __restrict__ vp) {
  constexpr int TN = 64;
  constexpr int LDS = D + 8;  // padded row: ldmatrix rows land in distinct banks
  constexpr int KSTEPS = D / 16;
  constexpr int DBLK = D / 8;
  constexpr int CH = D / 8;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  __nv_bfloat16* sK = reinterpret_cast<__nv_bfloat16*>(smem_raw);
  __nv_bfloat16* sV = sK + 2 * TN * LDS;

  const PadWorkItem it = plan_items(p)[blockIdx.x];
  const int R = it.n_events * p.group;
  const int row0 = blockIdx.y * 64;
  if (row0 >= R) return;
  const int kvh = it.kvh;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, t4 = lane & 3;

  const int rlo = row0 + warp * 16 + g, rhi = rlo + 8;
  GMask g_lo{0, 0, -1}, g_hi{0, 0, -1};
  if (p.g_self) {
    if (rlo < R) {
      const PadEventDesc ev = plan_events(p)[it.first_event + rlo / p.group];
      g_lo = g_mask_of(p, plan_videos(p)[ev.video], ev);
    }
    if (rhi < R) {
      const PadEventDesc ev = plan_events(p)[it.first_event + rhi / p.group];
      g_hi = g_mask_of(p, plan_videos(p)[ev.video], ev);
    }
  }
  uint32_t qa[KSTEPS][4];
  {
    const __nv_bfloat16* ql = rlo < R ? q_row(p, it.first_event, q, kvh, rlo) : nullptr;
    const __nv_bfloat16* qh = rhi < R ? q_row(p, it.first_event, q, kvh, rhi) : nullptr;
    if (p.rope_cs != nullptr) {
      const float* cl = ql ? p.rope_cs + (size_t)plan_events(p)[it.first_event + rlo / p.group].pos * D : nullptr;
      const float* ch = qh ? p.rope_cs + (size_t)plan_events(p)[it.first_event + rhi / p.group].pos * D : nullptr;
#pragma unroll
      for (int kk = 0; kk < KSTEPS; ++kk) {
        const int c = kk * 16 + 2 * t4;
        qa[kk][0] = ql ? rope_pair(ql, D, c, cl) : 0u;
        qa[kk][1] = qh ? rope_pair(qh, D, c, ch) : 0u;
        qa[kk][2] = ql ? rope_pair(ql, D, c + 8, cl) : 0u;
        qa[kk][3] = qh ? rope_pair(qh, D, c + 8, ch) : 0u;
      }
    } else {
#pragma unroll
      for (int kk = 0; kk < KSTEPS; ++kk) {
        const int c = kk * 16 + 2 * t4;
        qa[kk][0] = ql ? *reinterpret_cast<const uint32_t*>(ql + c) : 0u;
        qa[kk][1] = qh ? *reinterpret_cast<const uint32_t*>(qh + c) : 0u;
        qa[kk][2] = ql ? *reinterpret_cast<const uint32_t*>(ql + c + 8) : 0u;
        qa[kk][3] = qh ? *reinterpret_cast<const uint32_t*>(qh + c + 8) : 0u;
      }
    }
  }

  const size_t row_stride = (size_t)p.h_kv * D;
  // token t of the video's prefix (t relative to its start) is row (it.tok0 - it.tok_begin) + t
  const __nv_bfloat16* kbase = kp + (size_t)(it.tok0 - it.tok_begin) * row_stride + (size_t)kvh * D;
  const __nv_bfloat16* vbase = vp + (size_t)(it.tok0 - it.tok_begin) * row_stride + (size_t)kvh * D;
  const int ntiles = (it.tok_end - it.tok_begin + TN - 1) / TN;

  auto load_tile = [&](int tile, int stage) {
    const int base = it.tok_begin + tile * TN;
    for (int i = threadIdx.x; i < TN * CH; i += 128) {
      const int r = i / CH, c = i - (i / CH) * CH;
      const int tok = base + r;
      const bool ok = tok < it.tok_end;
      const size_t go = (size_t)(ok ? tok : it.tok_begin) * row_stride + c * 8;
      cp_async16(sK + (stage * TN + r) * LDS + c * 8, kbase + go, ok);
      cp_async16(sV + (stage * TN + r) * LDS + c * 8, vbase + go, ok);
    }
    cp_async_commit();
  };

  float o[DBLK][4];
#pragma unroll
  for (int i = 0; i < DBLK; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float m_lo = kNegInf, m_hi = kNegInf, l_lo = 0.f, l_hi = 0.f;

  load_tile(0, 0);
  for (int tile = 0; tile < ntiles; ++tile) {
    if (tile + 1 < ntiles) {
      load_tile(tile + 1, (tile + 1) & 1);
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    const __nv_bfloat16* tK = sK + (tile & 1) * TN * LDS;
    const __nv_bfloat16* tV = sV + (tile & 1) * TN * LDS;

    float s[TN / 8][4];
#pragma unroll
    for (int i = 0; i < TN / 8; ++i) s[i][0] = s[i][1] = s[i][2] = s[i][3] = 0.f;
#pragma unroll
    for (int nb2 = 0; nb2 < TN / 16; ++nb2) {
#pragma unroll
      for (int kk = 0; kk < KSTEPS; ++kk) {
        uint32_t b0, b1, b2, b3;
        ldsm_x4(b0, b1, b2, b3,
                tK + (nb2 * 16 + (lane >> 4) * 8 + (lane & 7)) * LDS + kk * 16 + ((lane >> 3) & 1) * 8);
        mma_bf16(s[2 * nb2], qa[kk], b0, b1);
        mma_bf16(s[2 * nb2 + 1], qa[kk], b2, b3);
      }
    }

    const int tb = it.tok_begin + tile * TN;   // prefix token of column 0
    const int valid = it.tok_end - tb;
    float mx_lo = kNegInf, mx_hi = kNegInf;
#pragma unroll
    for (int nb = 0; nb < TN / 8; ++nb) {
      const int c0 = nb * 8 + 2 * t4;
      s[nb][0] = c0 < valid && g_visible(g_lo, tb + c0) ? s[nb][0] * p.scale_log2 : kNegInf;
      s[nb][1] = c0 + 1 < valid && g_visible(g_lo, tb + c0 + 1) ? s[nb][1] * p.scale_log2 : kNegInf;
      s[nb][2] = c0 < valid && g_visible(g_hi, tb + c0) ? s[nb][2] * p.scale_log2 : kNegInf;
      s[nb][3] = c0 + 1 < valid && g_visible(g_hi, tb + c0 + 1) ? s[nb][3] * p.scale_log2 : kNegInf;
      mx_lo = fmaxf(mx_lo, fmaxf(s[nb][0], s[nb][1]));
      mx_hi = fmaxf(mx_hi, fmaxf(s[nb][2], s[nb][3]));
    }
    mx_lo = fmaxf(mx_lo, __shfl_xor_sync(0xffffffffu, mx_lo, 1));
    mx_lo = fmaxf(mx_lo, __shfl_xor_sync(0xffffffffu, mx_lo, 2));
    mx_hi = fmaxf(mx_hi, __shfl_xor_sync(0xffffffffu, mx_hi, 1));
    mx_hi = fmaxf(mx_hi, __shfl_xor_sync(0xffffffffu, mx_hi, 2));
    const float mn_lo = fmaxf(m_lo, mx_lo), mn_hi = fmaxf(m_hi, mx_hi);
    // -inf only while every token so far was hidden by the self G-token mask
    const float mb_lo = mn_lo == kNegInf ? 0.f : mn_lo, mb_hi = mn_hi == kNegInf ? 0.f : mn_hi;
    const float a_lo = ex2(m_lo - mb_lo), a_hi = ex2(m_hi - mb_hi);
    m_lo = mn_lo;
    m_hi = mn_hi;
    float rs_lo = 0.f, rs_hi = 0.f;
#pragma unroll
    for (int nb = 0; nb < TN / 8; ++nb) {
      s[nb][0] = ex2(s[nb][0] - mb_lo);
      s[nb][1] = ex2(s[nb][1] - mb_lo);
      s[nb][2] = ex2(s[nb][2] - mb_hi);
      s[nb][3] = ex2(s[nb][3] - mb_hi);
      rs_lo += s[nb][0] + s[nb][1];
      rs_hi += s[nb][2] + s[nb][3];
    }
    l_lo = l_lo * a_lo + rs_lo;
    l_hi = l_hi * a_hi + rs_hi;
#pragma unroll
    for (int db = 0; db < DBLK; ++db) {
      o[db][0] *= a_lo;
      o[db][1] *= a_lo;
      o[db][2] *= a_hi;
      o[db][3] *= a_hi;
    }

#pragma unroll
    for (int ks = 0; ks < TN / 16; ++ks) {
      uint32_t pa[4];
      pa[0] = pack_bf16(s[2 * ks][0], s[2 * ks][1]);
      pa[1] = pack_bf16(s[2 * ks][2], s[2 * ks][3]);
      pa[2] = pack_bf16(s[2 * ks + 1][0], s[2 * ks + 1][1]);
      pa[3] = pack_bf16(s[2 * ks + 1][2], s[2 * ks + 1][3]);
#pragma unroll
      for (int db2 = 0; db2 < DBLK / 2; ++db2) {
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(b0, b1, b2, b3,
                  tV + (ks * 16 + ((lane >> 3) & 1) * 8 + (lane & 7)) * LDS + (2 * db2 + (lane >> 4)) * 8);
        mma_bf16(o[2 * db2], pa, b0, b1);
        mma_bf16(o[2 * db2 + 1], pa, b2, b3);
      }
    }
    __syncthreads();
  }

  l_lo += __shfl_xor_sync(0xffffffffu, l_lo, 1);
  l_lo += __shfl_xor_sync(0xffffffffu, l_lo, 2);
  l_hi += __shfl_xor_sync(0xffffffffu, l_hi, 1);
  l_hi += __shfl_xor_sync(0xffffffffu, l_hi, 2);
  if (rlo < R) {
    const int64_t pr = (int64_t)it.part_row0 + rlo;
    if (t4 == 0) p.part_ml[pr] = make_float2(m_lo, l_lo);
    float* dst = p.part_o + pr * D;
#pragma unroll
    for (int db = 0; db < DBLK; ++db)
      *reinterpret_cast<float2*>(dst + db * 8 + 2 * t4) = make_float2(o[db][0], o[db][1]);
  }
  if (rhi < R) {
    const int64_t pr = (int64_t)it.part_row0 + rhi;
    if (t4 == 0) p.part_ml[pr] = make_float2(m_hi, l_hi);
    float* dst = p.part_o + pr * D;
#pragma unroll
    for (int db = 0; db < DBLK; ++db)
      *reinterpret_cast<float2*>(dst + db * 8 + 2 * t4) = make_float2(o[db][2], o[db][3]);
  }
}

// ---------------------------------------------------------------------------
// a4 + a5: one CTA (256 threads) per (event, kv-head); the task itself is
// bm::run_task (pad_branch_merge.cuh).  Launched after the prefix pass with
// programmatic dependent launch: its griddepcontrol.wait covers the prefix grid, so the
// split partials are complete once it returns.
// ---------------------------------------------------------------------------
// NW warps per task: 8 (two CTAs per SM) by default, 4 (three per SM) when the step has more
// than two waves of tasks, so that more of its latency-bound tasks are in flight at once.
template <int D, bool ROPE, int CAUSAL, int NW>
__global__ void __launch_bounds__(32 * NW, NW == bm::kWarps ? 2 : 3) branch_merge_kernel(const __grid_constant__ KParams p,
                                                                    const __nv_bfloat16* __restrict__ q,
                                                                    const __nv_bfloat16* __restrict__ kpool,
                                                                    const __nv_bfloat16* __restrict__ vpool,
                                                                    void* __restrict__ out,
                                                                    float* __restrict__ lse,
                                                                    int sch) {
  extern __shared__ __align__(16) unsigned char bm_raw[];
  // The grid after this one may be scheduled now: in a one-call loop it is the next step's
  // prefix kernel, which waits for this grid before it touches anything (an append kernel
  // after it is launched without programmatic serialisation and waits in any case).
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int e = blockIdx.x / p.h_kv;
  const int kvh = blockIdx.x - e * p.h_kv;
  bm::run_task<D, ROPE, CAUSAL, NW>(p, q, kpool, vpool, out, lse, e, kvh, (int)threadIdx.x, bm_raw, sch,
                                     bm::SyncCta{}, true, [] { return true; });
}

// Step inputs from page-locked, device-mapped host memory into device memory (the
// mapped-host-I/O form of pad_step_run_host): up to three 16-byte-aligned segments, read
// by the SMs over the host link.  It is launched so that it may start while the grid ahead
// still runs: each thread first loads up to kHeld pieces of every segment from host memory
// (the slow part), then waits for the grid ahead (which may still read these device
// buffers) before it stores anything.  It releases its dependents at entry; the step's first
// kernel waits for its completion before reading q.
struct HostInArgs {
  const uint4* src[3];
  uint4* dst[3];
  int64_t n16[3];
};
constexpr int kHostInHeld = 4;
__global__ void __launch_bounds__(256) host_in_kernel(const __grid_constant__ HostInArgs a) {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int64_t t0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  uint4 v[3][kHostInHeld];
#pragma unroll
  for (int k = 0; k < 3; ++k)
#pragma unroll
    for (int j = 0; j < kHostInHeld; ++j) {
      const int64_t i = t0 + j * stride;
      if (i < a.n16[k]) v[k][j] = a.src[k][i];
    }
  asm volatile("griddepcontrol.wait;" ::: "memory");
#pragma unroll
  for (int k = 0; k < 3; ++k) {
#pragma unroll
    for (int j = 0; j < kHostInHeld; ++j) {
      const int64_t i = t0 + j * stride;
      if (i < a.n16[k]) a.dst[k][i] = v[k][j];
    }
    // pieces past what a thread holds (inputs larger than the grid x kHostInHeld pieces)
    for (int64_t i = t0 + kHostInHeld * stride; i < a.n16[k]; i += stride) a.dst[k][i] = a.src[k][i];
  }
}

}  // namespace

cudaError_t launch_host_in(const void* const* src, void* const* dst, const size_t* bytes, int n, int sms,
                           cudaStream_t s) {
  if (n < 0 || n > 3) return cudaErrorInvalidValue;
  HostInArgs a{};
  int64_t largest = 0;
  for (int k = 0; k < n; ++k) {
    if ((bytes[k] & 15u) || (reinterpret_cast<uintptr_t>(src[k]) & 15u) || (reinterpret_cast<uintptr_t>(dst[k]) & 15u))
      return cudaErrorInvalidValue;
    a.src[k] = static_cast<const uint4*>(src[k]);
    a.dst[k] = static_cast<uint4*>(dst[k]);
    a.n16[k] = (int64_t)(bytes[k] >> 4);
    largest = std::max(largest, a.n16[k]);
  }
  if (largest == 0) return cudaSuccess;
  // enough threads that each holds at most kHostInHeld pieces of the largest segment,
  // at most one CTA of 256 per SM
  const int64_t per_cta = 256 * kHostInHeld;
  const int64_t blocks = std::min<int64_t>(std::max(1, sms), (largest + per_cta - 1) / per_cta);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)blocks);
  cfg.blockDim = dim3(256);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, host_in_kernel, a);
}

cudaError_t launch_append(const KParams& p, const void* k_new, const void* v_new, void* k_pool,
                          void* v_pool, cudaStream_t s) {
  const int total = p.n_events * p.h_kv * (p.head_dim / 8);
  if (total == 0) return cudaSuccess;
  const int bs = 256;
  append_kernel<<<(total + bs - 1) / bs, bs, 0, s>>>(
      p, static_cast<const uint4*>(k_new), static_cast<const uint4*>(v_new),
      static_cast<uint4*>(k_pool), static_cast<uint4*>(v_pool));
  return cudaGetLastError();
}

cudaError_t launch_prefix_simt(const KParams& p, int max_rows, const void* q, const void* kp,
                               const void* vp, cudaStream_t s) {
  if (p.n_items == 0) return cudaSuccess;
  auto Q = static_cast<const __nv_bfloat16*>(q);
  auto K = static_cast<const __nv_bfloat16*>(kp);
  auto V = static_cast<const __nv_bfloat16*>(vp);
  dim3 grid(p.n_items);
  if (p.head_dim == 128) {
    if (max_rows <= 8)
      prefix_simt_kernel<128, 8><<<grid, 256, 0, s>>>(p, Q, K, V);
    else
      prefix_simt_kernel<128, 16><<<grid, 256, 0, s>>>(p, Q, K, V);
  } else {
    if (max_rows <= 8)
      prefix_simt_kernel<64, 8><<<grid, 256, 0, s>>>(p, Q, K, V);
    else
      prefix_simt_kernel<64, 16><<<grid, 256, 0, s>>>(p, Q, K, V);
  }
  return cudaGetLastError();
}

template <int D>
static cudaError_t launch_mma_d(const KParams& p, int max_rows, const void* q, const void* kp,
                                const void* vp, cudaStream_t s) {
  constexpr int TN = 64, LDS = D + 8;
  const size_t smem = 2ull * 2 * TN * LDS * sizeof(__nv_bfloat16);
  static bool configured[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64 && !configured[dev]) {
    cudaError_t e = cudaFuncSetAttribute(prefix_mma_kernel<D>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    configured[dev] = true;
  }
  dim3 grid(p.n_items, (max_rows + 63) / 64);
  prefix_mma_kernel<D><<<grid, 128, smem, s>>>(p, static_cast<const __nv_bfloat16*>(q),
                                               static_cast<const __nv_bfloat16*>(kp),
                                               static_cast<const __nv_bfloat16*>(vp));
  return cudaGetLastError();
}

cudaError_t launch_prefix_mma(const KParams& p, int max_rows, const void* q, const void* kp,
                              const void* vp, cudaStream_t s) {
  if (p.n_items == 0) return cudaSuccess;
  if (p.head_dim == 128) return launch_mma_d<128>(p, max_rows, q, kp, vp, s);
  return launch_mma_d<64>(p, max_rows, q, kp, vp, s);
}

// Split partials merged per staged chunk: as many as a shared-memory budget allows next to
// the branch staging.
template <int D, int NW = bm::kWarps>
int bm_chunk(const KParams& p, size_t budget) {
  const int G = p.group;
  const size_t fixed =
      bm::align16(sizeof(bm::Head<D>)) + bm::kv_bytes<D, NW>(bm::round_keys(p.branch_rows, NW), G) + 16;
  const size_t per_split = (size_t)G * D * sizeof(float) + sizeof(float2);
  int sch = fixed + per_split <= budget ? (int)((budget - fixed) / per_split) : 1;
  if (p.max_splits > 0 && sch > p.max_splits) sch = p.max_splits;
  return sch < 1 ? 1 : (sch > bm::kMaxChunk ? bm::kMaxChunk : sch);
}
// The standalone kernel: a grid of more CTAs than SMs keeps two per SM (8 warps each), one
// of more than two waves three (4 warps each).
inline bool bm_narrow(const KParams& p) { return (int64_t)p.n_events * p.h_kv > 2 * (int64_t)p.n_sms; }
inline size_t n_cta_budget(const KParams& p) {
  if (bm_narrow(p)) return 74 * 1024;
  return p.n_events * p.h_kv > p.n_sms ? 110 * 1024 : 200 * 1024;
}

template <int D, int NW>
static cudaError_t launch_bm_nw(const KParams& p, const void* q, const void* k_pool, const void* v_pool,
                                void* out, float* lse, bool pdl, cudaStream_t s) {
  const int G = p.group;
  const int nkr = p.branch_rows;
  if (nkr <= 0 || nkr > bm::kKeys || nkr % 16 != 0) return cudaErrorInvalidValue;
  const int sch = bm_chunk<D, NW>(p, n_cta_budget(p));
  const size_t smem = bm::smem_bytes<D, NW>(nkr, G, sch);
  constexpr int kMaxSmem = 227 * 1024;
  if (smem > (size_t)kMaxSmem) return cudaErrorInvalidValue;
  static bool configured[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64 && !configured[dev]) {
    for (auto fn : {branch_merge_kernel<D, false, 0, NW>, branch_merge_kernel<D, true, 0, NW>,
                    branch_merge_kernel<D, false, 1, NW>, branch_merge_kernel<D, true, 1, NW>}) {
      cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, kMaxSmem);
      if (e != cudaSuccess) return e;
    }
    configured[dev] = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.n_events * p.h_kv);
  cfg.blockDim = dim3(32 * NW);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  auto fn = p.causal ? (p.rope_cs != nullptr ? branch_merge_kernel<D, true, 1, NW> : branch_merge_kernel<D, false, 1, NW>)
                     : (p.rope_cs != nullptr ? branch_merge_kernel<D, true, 0, NW> : branch_merge_kernel<D, false, 0, NW>);
  return cudaLaunchKernelEx(&cfg, fn, p, static_cast<const __nv_bfloat16*>(q),
                            static_cast<const __nv_bfloat16*>(k_pool), static_cast<const __nv_bfloat16*>(v_pool),
                            out, lse, sch);
}
template <int D>
static cudaError_t launch_bm(const KParams& p, const void* q, const void* k_pool, const void* v_pool,
                             void* out, float* lse, bool pdl, cudaStream_t s) {
  return bm_narrow(p) ? launch_bm_nw<D, 4>(p, q, k_pool, v_pool, out, lse, pdl, s)
                      : launch_bm_nw<D, bm::kWarps>(p, q, k_pool, v_pool, out, lse, pdl, s);
}

cudaError_t launch_branch_merge(const KParams& p, const void* q, const void* k_pool,
                                const void* v_pool, void* out, float* lse, bool pdl, cudaStream_t s) {
  if (p.n_events == 0) return cudaSuccess;
  if (p.head_dim == 128) return launch_bm<128>(p, q, k_pool, v_pool, out, lse, pdl, s);
  return launch_bm<64>(p, q, k_pool, v_pool, out, lse, pdl, s);
}

}  // namespace pad
