// Kernels of one event-factorized decode step (Sec. 3.4, Eq. 3):
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
  // the shared-prefix pass launched after this kernel reads nothing it writes
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int chunks = p.head_dim / 8;
  const int per_event = p.h_kv * chunks;
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
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
  k_pool[dst] = k_new[src];
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

  const PadWorkItem it = plan_items(p)[blockIdx.x];
  const int R = it.n_events * p.group;
  const int kvh = it.kvh;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  for (int i = threadIdx.x; i < MAXR * D; i += blockDim.x) {
    int r = i / D, d = i - r * D;
    float v = 0.f;
    if (r < R) v = __bfloat162float(q_row(p, it.first_event, q, kvh, r)[d]);
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
        float sv = valid ? s[r] * p.scale_log2 : kNegInf;
        float mn = fmaxf(m[r], warp_max(sv));       // finite: lane 0's token is valid
        float alpha = ex2(m[r] - mn);
        float pr = ex2(sv - mn);
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
  uint32_t qa[KSTEPS][4];
  {
    const __nv_bfloat16* ql = rlo < R ? q_row(p, it.first_event, q, kvh, rlo) : nullptr;
    const __nv_bfloat16* qh = rhi < R ? q_row(p, it.first_event, q, kvh, rhi) : nullptr;
#pragma unroll
    for (int kk = 0; kk < KSTEPS; ++kk) {
      const int c = kk * 16 + 2 * t4;
      qa[kk][0] = ql ? *reinterpret_cast<const uint32_t*>(ql + c) : 0u;
      qa[kk][1] = qh ? *reinterpret_cast<const uint32_t*>(qh + c) : 0u;
      qa[kk][2] = ql ? *reinterpret_cast<const uint32_t*>(ql + c + 8) : 0u;
      qa[kk][3] = qh ? *reinterpret_cast<const uint32_t*>(qh + c + 8) : 0u;
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

    const int valid = it.tok_end - (it.tok_begin + tile * TN);
    float mx_lo = kNegInf, mx_hi = kNegInf;
#pragma unroll
    for (int nb = 0; nb < TN / 8; ++nb) {
      const int c0 = nb * 8 + 2 * t4;
      s[nb][0] = c0 < valid ? s[nb][0] * p.scale_log2 : kNegInf;
      s[nb][1] = c0 + 1 < valid ? s[nb][1] * p.scale_log2 : kNegInf;
      s[nb][2] = c0 < valid ? s[nb][2] * p.scale_log2 : kNegInf;
      s[nb][3] = c0 + 1 < valid ? s[nb][3] * p.scale_log2 : kNegInf;
      mx_lo = fmaxf(mx_lo, fmaxf(s[nb][0], s[nb][1]));
      mx_hi = fmaxf(mx_hi, fmaxf(s[nb][2], s[nb][3]));
    }
    mx_lo = fmaxf(mx_lo, __shfl_xor_sync(0xffffffffu, mx_lo, 1));
    mx_lo = fmaxf(mx_lo, __shfl_xor_sync(0xffffffffu, mx_lo, 2));
    mx_hi = fmaxf(mx_hi, __shfl_xor_sync(0xffffffffu, mx_hi, 1));
    mx_hi = fmaxf(mx_hi, __shfl_xor_sync(0xffffffffu, mx_hi, 2));
    const float mn_lo = fmaxf(m_lo, mx_lo), mn_hi = fmaxf(m_hi, mx_hi);  // finite (valid >= 1)
    const float a_lo = ex2(m_lo - mn_lo), a_hi = ex2(m_hi - mn_hi);
    m_lo = mn_lo;
    m_hi = mn_hi;
    float rs_lo = 0.f, rs_hi = 0.f;
#pragma unroll
    for (int nb = 0; nb < TN / 8; ++nb) {
      s[nb][0] = ex2(s[nb][0] - mn_lo);
      s[nb][1] = ex2(s[nb][1] - mn_lo);
      s[nb][2] = ex2(s[nb][2] - mn_hi);
      s[nb][3] = ex2(s[nb][3] - mn_hi);
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
// a4 + a5: one CTA (256 threads, 8 warps) per (event, kv-head).
//   a4, the own-branch part of the mask of Sec. 3.4: the branch's keys 0..len, its
//   private tokens and the one appended at this step, staged in rounds of kBmKeys (K and
//   V rows through the page table, cp.async); each warp takes 16 of a round's keys and
//   keeps a flash-attention state held in registers in the manner of the warp-level MMA
//   kernels (the G <= 16 query rows form one m16 tile, S = Q K^T, online softmax on the
//   accumulators in base 2, O += P V with P re-packed from the S accumulators).
//   a5: the eight warp states and the prefix splits' partial states are merged by
//   log-sum-exp: M = max of the maxima, every state weighted by 2^(m - M).
//   The CTA starts as the shared-prefix pass's CTAs retire.  Before griddepcontrol.wait it
//   stages what the grids ahead do not write: Q rows, the branch's page ids and the K/V
//   rows of its earlier keys.  After it, in one round trip: key `len` (written by this
//   step's append), the splits' (m, l) pairs and (one bulk copy per split, on an
//   mbarrier) their fp32 O rows.
// ---------------------------------------------------------------------------
constexpr int kBmThreads = 256;
constexpr int kBmWarps = kBmThreads / 32;
constexpr int kBmKeys = 16 * kBmWarps;        // branch keys staged per round
constexpr int kBmMaxChunk = 64;               // prefix splits merged per staged chunk
constexpr unsigned long long kBmWaitNs = 1000000000ull;  // one second per bounded wait

__host__ __device__ constexpr size_t bm_align16(size_t x) { return (x + 15) / 16 * 16; }

// Shared memory: this head, then three regions sized per launch (16-byte aligned):
//   kv   K rows [nkr][LD] and V rows [nkr][LD] of a round (nkr = KParams::branch_rows);
//        after the branch pass the warps' O rows, fp32 [warp][G][D]
//   ml   the splits' (m, l) pairs of a chunk, [G][sch]
//   po   the splits' O rows of a chunk, fp32 [sch][G][D]
template <int D>
struct BmHead {
  static constexpr int LD = D + 8;            // padded bf16 row: ldmatrix rows in distinct banks
  __nv_bfloat16 q[16][LD];
  int page[kBmKeys];
  float wm[kBmWarps][16], wl[kBmWarps][16];   // each warp's branch state per row
  float sc[16][kBmMaxChunk];                  // state weights 2^(m - M)
  alignas(16) float ob[16][D];                // merged numerator (read as float4)
  float M[16], L[16], a[16];
  unsigned long long bar;                     // completion of a chunk's bulk copies
};
__host__ __device__ constexpr size_t bm_max(size_t a, size_t b) { return a > b ? a : b; }
template <int D>
__host__ __device__ constexpr size_t bm_kv_bytes(int nkr, int G) {
  return bm_align16(bm_max((size_t)2 * nkr * BmHead<D>::LD * 2, (size_t)kBmWarps * G * D * 4));
}
template <int D>
__host__ __device__ constexpr size_t bm_smem_bytes(int nkr, int G, int sch) {
  return bm_align16(sizeof(BmHead<D>)) + bm_kv_bytes<D>(nkr, G) + bm_align16((size_t)G * sch * 8) +
         (size_t)sch * G * D * 4;
}

__device__ __forceinline__ uint32_t bm_smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ unsigned long long bm_globaltimer() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
// Bounded wait for the phase of the given parity of the chunk barrier; false = gave up.
__device__ __forceinline__ bool bm_wait(unsigned long long* bar, uint32_t parity) {
  const unsigned long long t0 = bm_globaltimer();
  for (;;) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
        " selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(bm_smem_u32(bar)), "r"(parity)
        : "memory");
    if (ok) return true;
    if (bm_globaltimer() - t0 > kBmWaitNs) return false;
  }
}
__device__ __forceinline__ void cp_async8(void* smem, const void* gmem) {
  unsigned s = static_cast<unsigned>(__cvta_generic_to_shared(smem));
  asm volatile("cp.async.ca.shared.global [%0], [%1], 8;\n" ::"r"(s), "l"(gmem));
}

template <int D>
__global__ void __launch_bounds__(kBmThreads) branch_merge_kernel(const __grid_constant__ KParams p,
                                                                  const __nv_bfloat16* __restrict__ q,
                                                                  const __nv_bfloat16* __restrict__ kpool,
                                                                  const __nv_bfloat16* __restrict__ vpool,
                                                                  void* __restrict__ out,
                                                                  float* __restrict__ lse,
                                                                  int sch) {
  constexpr int NT = kBmThreads;
  constexpr int CH = D / 8;                   // 16-byte pieces of a bf16 row
  constexpr int KS = D / 16;                  // k-steps of S = Q K^T
  constexpr int OT = D / 8;                   // n8 tiles of O
  constexpr int LD = BmHead<D>::LD;
  extern __shared__ __align__(16) unsigned char bm_raw[];
  BmHead<D>& S = *reinterpret_cast<BmHead<D>*>(bm_raw);
  const int G = p.group;
  const int nkr = p.branch_rows;              // keys per round (multiple of 16, <= kBmKeys)
  unsigned char* kv_raw = bm_raw + bm_align16(sizeof(BmHead<D>));
  __nv_bfloat16 (*sK)[LD] = reinterpret_cast<__nv_bfloat16 (*)[LD]>(kv_raw);
  __nv_bfloat16 (*sV)[LD] = reinterpret_cast<__nv_bfloat16 (*)[LD]>(kv_raw + (size_t)nkr * LD * 2);
  float* wo = reinterpret_cast<float*>(kv_raw);  // [warp][G][d] after the branch pass
  float2* sml = reinterpret_cast<float2*>(kv_raw + bm_kv_bytes<D>(nkr, G));
  float* spo = reinterpret_cast<float*>(reinterpret_cast<unsigned char*>(sml) + bm_align16((size_t)G * sch * 8));

  const int e = blockIdx.x / p.h_kv;
  const int kvh = blockIdx.x - e * p.h_kv;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int gq = lane >> 2, t4 = lane & 3;
  const PadEventDesc ev = plan_events(p)[e];
  const PadVideoDesc vd = plan_videos(p)[ev.video];
  const int R = vd.n_events * G;
  const int ns = vd.n_splits;
  const int rbase = ev.local * G;
  const int len = ev.len;                     // keys before this step; key `len` is this step's
  const int nk = len + 1;
  const int ps = p.page_size;
  const int32_t* ptab = p.page_table + (size_t)e * p.max_pages;

  // page of key c0 + tid: the page this step took for key `len`, else the table's entry
  // (written by an earlier step)
  auto page_of = [&](int key) -> int {
    const int pi = key / ps;
    int page = (pi == len / ps && ev.new_page >= 0) ? ev.new_page : ptab[pi];
    if (page < 0 || page >= p.n_pages) {
      pad_set_error(p.header, p.gen, PAD_ERR_DEVICE_BOUNDS, e, pi, page);
      page = -1;
    }
    return page;
  };
  // Before the wait: Q rows, the first round's page ids (key `len`'s page is the one this
  // step took, else the table's entry of an earlier step) and its K/V rows except key
  // `len`, which this step's append writes
  const int nv0 = min(nkr, nk);
  if (tid < nkr) S.page[tid] = tid < nv0 ? page_of(tid) : -1;
  if (tid == 0) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(bm_smem_u32(&S.bar)) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  for (int i = tid; i < 16 * CH; i += NT) {
    const int g = i / CH, c = i - (i / CH) * CH;
    const bool in = g < G;
    cp_async16(&S.q[g][c * 8], q + ((size_t)e * p.h_q + kvh * G + (in ? g : 0)) * D + c * 8, in);
  }
  for (int i = tid; i < G * D; i += NT) S.ob[i / D][i % D] = 0.f;
  if (tid < 16) {
    S.M[tid] = kNegInf;
    S.L[tid] = 0.f;
  }
  __syncthreads();
  auto stage_keys = [&](int r0, int nv, int k_lo, int k_hi) {  // rows k_lo..k_hi-1 of the round
    for (int i = tid; i < (k_hi - k_lo) * CH; i += NT) {
      const int k = k_lo + i / CH, c = i - (i / CH) * CH;
      const int pg = k < nv ? S.page[k] : -1;
      const bool in = pg >= 0;
      const size_t off = (((size_t)(in ? pg : 0) * p.h_kv + kvh) * ps + ((r0 + k) % ps)) * D + c * 8;
      cp_async16(&sK[k][c * 8], kpool + off, in);
      cp_async16(&sV[k][c * 8], vpool + off, in);
    }
  };
  const int nv0_16 = (nv0 + 15) & ~15;
  const bool len_in_first = len < nkr;
  // rows 0..nv0_16-1 except key `len` (rows past nv0 are zero-filled)
  if (len_in_first) {
    stage_keys(0, nv0, 0, len);
    stage_keys(0, nv0, len + 1, nv0_16);
  } else {
    stage_keys(0, nv0, 0, nv0_16);
  }
  cp_async_commit();

  // ---------------- after the shared-prefix pass (and, through it, the append) completed
  asm volatile("griddepcontrol.wait;" ::: "memory");
  if (len_in_first) stage_keys(0, nv0, len, len + 1);
  cp_async_commit();                          // this round's keys

  const uint32_t bytes_per_split = (uint32_t)(G * D * sizeof(float));
  // the splits' O rows (bulk copies) and (m, l) pairs of chunk [s0, s0 + nch)
  auto stage_chunk = [&](int s0, int nch) {
    if (tid == NT - 1) {
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bm_smem_u32(&S.bar)),
                   "r"(bytes_per_split * (uint32_t)nch)
                   : "memory");
      for (int sl = 0; sl < nch; ++sl)
        asm volatile(
            "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                bm_smem_u32(spo + (size_t)sl * G * D)),
            "l"(p.part_o + part_row(vd, kvh, s0 + sl, R, rbase) * D), "r"(bytes_per_split),
            "r"(bm_smem_u32(&S.bar))
            : "memory");
    }
    for (int i = tid; i < G * nch; i += NT) {
      const int g = i / nch, sl = i - g * nch;
      cp_async8(&sml[g * sch + sl], &p.part_ml[part_row(vd, kvh, s0 + sl, R, rbase + g)]);
    }
  };
  if (ns > 0) stage_chunk(0, min(sch, ns));
  cp_async_commit();                          // the first chunk's (m, l) pairs, waited for in a5

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
      if (tid < nkr) S.page[tid] = tid < nv ? page_of(r0 + tid) : -1;
      __syncthreads();
      stage_keys(r0, nv, 0, (nv + 15) & ~15);
      cp_async_commit();
      cp_async_wait<0>();
    } else {
      cp_async_wait<1>();                     // all but the (m, l) group
    }
    __syncthreads();
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
    __syncthreads();                          // the next round (or the O rows below) overwrite k / v
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
  __syncthreads();

  // ---------------- a5: the warp states, then the prefix splits in chunks of `sch`
  // (M, L, numerator) = log-sum-exp merge of the warps' states: one warp per row
  for (int g = warp; g < G; g += kBmWarps) {
    const float mw = lane < kBmWarps ? S.wm[lane][g] : kNegInf;
    float mx = warp_max(mw);
    if (mx == kNegInf) mx = 0.f;              // no key of the branch passed its bounds check
    const float wgt = lane < kBmWarps ? ex2(mw - mx) : 0.f;
    const float sum = warp_sum(lane < kBmWarps ? S.wl[lane][g] * wgt : 0.f);
    if (lane < kBmWarps) S.sc[g][lane] = wgt;
    if (lane == 0) {
      S.M[g] = mx;
      S.L[g] = sum;
    }
  }
  __syncthreads();
  constexpr int D4 = D / 4;
  for (int i = tid; i < G * D4; i += NT) {
    const int g = i / D4, d4 = i - g * D4;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int w = 0; w < kBmWarps; ++w) {
      const float c = S.sc[g][w];
      const float4 v = reinterpret_cast<const float4*>(wo)[(w * G + g) * D4 + d4];
      acc.x = fmaf(c, v.x, acc.x);
      acc.y = fmaf(c, v.y, acc.y);
      acc.z = fmaf(c, v.z, acc.z);
      acc.w = fmaf(c, v.w, acc.w);
    }
    reinterpret_cast<float4*>(&S.ob[g][0])[d4] = acc;
  }

  bool staged_ok = true;
  for (int s0 = 0, chunk = 0; s0 < ns; s0 += sch, ++chunk) {
    const int nch = min(sch, ns - s0);
    if (s0 > 0) {
      __syncthreads();                        // the previous chunk's rows are consumed
      stage_chunk(s0, nch);
    }
    cp_async_commit();
    cp_async_wait<0>();                       // the (m, l) pairs
    __syncthreads();
    // row statistics, one warp per row, lanes over splits
    for (int g = warp; g < G; g += kBmWarps) {
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
    if (!bm_wait(&S.bar, (uint32_t)(chunk & 1))) {
      staged_ok = false;
      if (tid == 0) pad_set_error(p.header, p.gen, PAD_ERR_DEVICE_TIMEOUT, e, -1, chunk);
    }
    if (!__syncthreads_and(staged_ok)) {
      // the copies must land before this CTA's shared memory is released
      bm_wait(&S.bar, (uint32_t)(chunk & 1));
      break;
    }
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
  __syncthreads();

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

}  // namespace

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

template <int D>
static cudaError_t launch_bm(const KParams& p, const void* q, const void* k_pool, const void* v_pool,
                             void* out, float* lse, bool pdl, cudaStream_t s) {
  const int G = p.group;
  const int nkr = p.branch_rows;
  if (nkr <= 0 || nkr > kBmKeys || nkr % 16 != 0) return cudaErrorInvalidValue;
  // Staged prefix partials: as many splits per chunk as a budget allows; a grid larger than
  // one wave keeps two CTAs per SM.
  const int n_cta = p.n_events * p.h_kv;
  const size_t budget = n_cta > p.n_sms ? 110 * 1024 : 200 * 1024;
  const size_t fixed = bm_align16(sizeof(BmHead<D>)) + bm_kv_bytes<D>(nkr, G) + 16;
  const size_t per_split = (size_t)G * D * sizeof(float) + sizeof(float2);
  int sch = fixed + per_split <= budget ? (int)((budget - fixed) / per_split) : 1;
  if (p.max_splits > 0 && sch > p.max_splits) sch = p.max_splits;
  sch = sch < 1 ? 1 : (sch > kBmMaxChunk ? kBmMaxChunk : sch);
  const size_t smem = bm_smem_bytes<D>(nkr, G, sch);
  constexpr int kMaxSmem = 227 * 1024;
  if (smem > (size_t)kMaxSmem) return cudaErrorInvalidValue;
  static bool configured[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64 && !configured[dev]) {
    cudaError_t e = cudaFuncSetAttribute(branch_merge_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         kMaxSmem);
    if (e != cudaSuccess) return e;
    configured[dev] = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.n_events * p.h_kv);
  cfg.blockDim = dim3(kBmThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, branch_merge_kernel<D>, p, static_cast<const __nv_bfloat16*>(q),
                            static_cast<const __nv_bfloat16*>(k_pool), static_cast<const __nv_bfloat16*>(v_pool),
                            out, lse, sch);
}

cudaError_t launch_branch_merge(const KParams& p, const void* q, const void* k_pool,
                                const void* v_pool, void* out, float* lse, bool pdl, cudaStream_t s) {
  if (p.n_events == 0) return cudaSuccess;
  if (p.head_dim == 128) return launch_bm<128>(p, q, k_pool, v_pool, out, lse, pdl, s);
  return launch_bm<64>(p, q, k_pool, v_pool, out, lse, pdl, s);
}

}  // namespace pad
