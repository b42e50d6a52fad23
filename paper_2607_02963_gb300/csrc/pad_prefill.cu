// Training / prefill forward attention under the full-sequence event-factorized mask
// (Sec. 3.4, Fig. 3): the sequence of one video is [shared prefix of S tokens (P, the
// planning tokens G^1..G^K, S) ; branch 1 ; ... ; branch E].  A prefix token attends
// causally within the prefix; a branch token attends to the whole prefix and causally to
// its own branch; no token attends to another branch.  The paper runs this mask through a
// generic masked attention and names the missing kernel as the cause of its extra training
// time; here it is block-sparse by construction.
//
// One CTA (4 warps, 64 query tokens, one q-head) walks only the keys its rows can see: the
// prefix up to its last row, then the keys from the start of its first row's branch to its
// last row (a tile spans at most a few branches).  Prefix tiles below the tile's first row
// need no mask; the diagonal and the branch tiles are masked per element.  Warp-level
// mma.sync m16n8k16 (bf16 in, fp32 accumulate), K/V tiles of 64 keys double-buffered with
// cp.async, online softmax in base 2; O and the LSE are written normalised, once.
#include <cuda_bf16.h>
#include <algorithm>
#include <cstdint>

#include "pad_branch_merge.cuh"
#include "pad_internal.h"

namespace pad {
namespace {

constexpr int kMaxBranches = 1024;
constexpr int kTN = 64;        // keys per tile
constexpr int kTM = 64;        // query tokens per CTA
constexpr int kThreads = 128;  // 4 warps x 16 rows

struct PrefillParams {
  int32_t n_tokens, prefix_len, n_branches;
  int32_t h_q, h_kv, group;
  float scale_log2;
  int32_t out_bf16;
  int32_t bstart[kMaxBranches + 1];  // branch b occupies [bstart[b], bstart[b + 1]); bstart[0] = prefix_len
};

// First token of the branch that holds token p (p >= prefix_len).
__device__ __forceinline__ int branch_start(const PrefillParams& pp, int p) {
  int lo = 0, hi = pp.n_branches - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (pp.bstart[mid] <= p) lo = mid; else hi = mid - 1;
  }
  return pp.bstart[lo];
}

// Key t visible to query token p (bs: p's branch start, or -1 for a prefix token).
__device__ __forceinline__ bool visible(int p, int bs, int S, int t) {
  return bs < 0 ? t <= p : (t < S || (t >= bs && t <= p));
}

template <int D>
__global__ void __launch_bounds__(kThreads) prefill_mma_kernel(const __grid_constant__ PrefillParams pp,
                                                               const __nv_bfloat16* __restrict__ q,
                                                               const __nv_bfloat16* __restrict__ k,
                                                               const __nv_bfloat16* __restrict__ v, void* __restrict__ out,
                                                               float* __restrict__ lse) {
  using namespace bm;
  constexpr int LDS = D + 8;  // padded row: ldmatrix rows land in distinct banks
  constexpr int KSTEPS = D / 16;
  constexpr int DBLK = D / 8;
  constexpr int CH = D / 8;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  __nv_bfloat16* sK = reinterpret_cast<__nv_bfloat16*>(smem_raw);
  __nv_bfloat16* sV = sK + 2 * kTN * LDS;

  const int N = pp.n_tokens, S = pp.prefix_len;
  const int p0 = blockIdx.x * kTM, h = blockIdx.y, kvh = h / pp.group;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, t4 = lane & 3;
  const int plo = p0 + warp * 16 + g, phi = plo + 8;
  const int bs_lo = plo >= S && plo < N ? branch_start(pp, plo) : -1;
  const int bs_hi = phi >= S && phi < N ? branch_start(pp, phi) : -1;

  uint32_t qa[KSTEPS][4];
  {
    const __nv_bfloat16* ql = plo < N ? q + ((size_t)plo * pp.h_q + h) * D : nullptr;
    const __nv_bfloat16* qh = phi < N ? q + ((size_t)phi * pp.h_q + h) * D : nullptr;
#pragma unroll
    for (int kk = 0; kk < KSTEPS; ++kk) {
      const int c = kk * 16 + 2 * t4;
      qa[kk][0] = ql ? *reinterpret_cast<const uint32_t*>(ql + c) : 0u;
      qa[kk][1] = qh ? *reinterpret_cast<const uint32_t*>(qh + c) : 0u;
      qa[kk][2] = ql ? *reinterpret_cast<const uint32_t*>(ql + c + 8) : 0u;
      qa[kk][3] = qh ? *reinterpret_cast<const uint32_t*>(qh + c + 8) : 0u;
    }
  }

  // key ranges: A = [0, a_end) of the prefix, B = [b_lo, b_end) of the branches
  const int last = min(p0 + kTM - 1, N - 1);
  const int a_end = min(S, last + 1);
  const int b_lo = last >= S ? branch_start(pp, max(p0, S)) : 0;
  const int b_end = last >= S ? last + 1 : 0;
  const int nA = (a_end + kTN - 1) / kTN, nB = (b_end - b_lo + kTN - 1) / kTN;
  const int ntiles = nA + nB;
  auto tile_range = [&](int i, int& tb, int& te) {
    if (i < nA) {
      tb = i * kTN;
      te = min(a_end, tb + kTN);
    } else {
      tb = b_lo + (i - nA) * kTN;
      te = min(b_end, tb + kTN);
    }
  };
  const size_t row_stride = (size_t)pp.h_kv * D;
  const __nv_bfloat16* kbase = k + (size_t)kvh * D;
  const __nv_bfloat16* vbase = v + (size_t)kvh * D;
  auto load_tile = [&](int i, int stage) {
    int tb, te;
    tile_range(i, tb, te);
    for (int j = threadIdx.x; j < kTN * CH; j += kThreads) {
      const int r = j / CH, c = j - (j / CH) * CH;
      const int tok = tb + r;
      const bool ok = tok < te;
      const size_t go = (size_t)(ok ? tok : tb) * row_stride + c * 8;
      cp_async16(sK + (stage * kTN + r) * LDS + c * 8, kbase + go, ok);
      cp_async16(sV + (stage * kTN + r) * LDS + c * 8, vbase + go, ok);
    }
    cp_async_commit();
  };

  float o[DBLK][4];
#pragma unroll
  for (int i = 0; i < DBLK; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float m_lo = kNegInf, m_hi = kNegInf, l_lo = 0.f, l_hi = 0.f;
  const float sl2 = pp.scale_log2;

  if (ntiles > 0) load_tile(0, 0);
  for (int i = 0; i < ntiles; ++i) {
    if (i + 1 < ntiles) {
      load_tile(i + 1, (i + 1) & 1);
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    const __nv_bfloat16* tK = sK + (i & 1) * kTN * LDS;
    const __nv_bfloat16* tV = sV + (i & 1) * kTN * LDS;
    int tb, te;
    tile_range(i, tb, te);

    float s[kTN / 8][4];
#pragma unroll
    for (int j = 0; j < kTN / 8; ++j) s[j][0] = s[j][1] = s[j][2] = s[j][3] = 0.f;
#pragma unroll
    for (int nb2 = 0; nb2 < kTN / 16; ++nb2) {
#pragma unroll
      for (int kk = 0; kk < KSTEPS; ++kk) {
        uint32_t b0, b1, b2, b3;
        ldsm_x4(b0, b1, b2, b3,
                tK + (nb2 * 16 + (lane >> 4) * 8 + (lane & 7)) * LDS + kk * 16 + ((lane >> 3) & 1) * 8);
        mma_bf16(s[2 * nb2], qa[kk], b0, b1);
        mma_bf16(s[2 * nb2 + 1], qa[kk], b2, b3);
      }
    }

    // prefix tiles wholly below the CTA's first token need no mask (all rows see them)
    const bool full = i < nA && te - tb == kTN && (p0 >= S || te - 1 <= p0) && last < N && p0 + kTM <= N;
    float mx_lo = kNegInf, mx_hi = kNegInf;
#pragma unroll
    for (int nb = 0; nb < kTN / 8; ++nb) {
      const int c0 = tb + nb * 8 + 2 * t4;
      if (full) {
        s[nb][0] *= sl2;
        s[nb][1] *= sl2;
        s[nb][2] *= sl2;
        s[nb][3] *= sl2;
      } else {
        s[nb][0] = c0 < te && plo < N && visible(plo, bs_lo, S, c0) ? s[nb][0] * sl2 : kNegInf;
        s[nb][1] = c0 + 1 < te && plo < N && visible(plo, bs_lo, S, c0 + 1) ? s[nb][1] * sl2 : kNegInf;
        s[nb][2] = c0 < te && phi < N && visible(phi, bs_hi, S, c0) ? s[nb][2] * sl2 : kNegInf;
        s[nb][3] = c0 + 1 < te && phi < N && visible(phi, bs_hi, S, c0 + 1) ? s[nb][3] * sl2 : kNegInf;
      }
      mx_lo = fmaxf(mx_lo, fmaxf(s[nb][0], s[nb][1]));
      mx_hi = fmaxf(mx_hi, fmaxf(s[nb][2], s[nb][3]));
    }
    mx_lo = fmaxf(mx_lo, __shfl_xor_sync(0xffffffffu, mx_lo, 1));
    mx_lo = fmaxf(mx_lo, __shfl_xor_sync(0xffffffffu, mx_lo, 2));
    mx_hi = fmaxf(mx_hi, __shfl_xor_sync(0xffffffffu, mx_hi, 1));
    mx_hi = fmaxf(mx_hi, __shfl_xor_sync(0xffffffffu, mx_hi, 2));
    const float mn_lo = fmaxf(m_lo, mx_lo), mn_hi = fmaxf(m_hi, mx_hi);
    // -inf only while a row has seen no visible key yet (exponent base 0 avoids NaN)
    const float mb_lo = mn_lo == kNegInf ? 0.f : mn_lo, mb_hi = mn_hi == kNegInf ? 0.f : mn_hi;
    const float a_lo = ex2(m_lo - mb_lo), a_hi = ex2(m_hi - mb_hi);
    m_lo = mn_lo;
    m_hi = mn_hi;
    float rs_lo = 0.f, rs_hi = 0.f;
#pragma unroll
    for (int nb = 0; nb < kTN / 8; ++nb) {
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
    for (int ks = 0; ks < kTN / 16; ++ks) {
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
  auto store = [&](int p, float m, float l, int half) {
    if (p >= N) return;
    const float inv = 1.0f / l;
    const size_t row = (size_t)p * pp.h_q + h;
#pragma unroll
    for (int db = 0; db < DBLK; ++db) {
      const float x0 = o[db][2 * half] * inv, x1 = o[db][2 * half + 1] * inv;
      const size_t oi = row * D + db * 8 + 2 * t4;
      if (pp.out_bf16)
        *reinterpret_cast<uint32_t*>(reinterpret_cast<__nv_bfloat16*>(out) + oi) = pack_bf16(x0, x1);
      else
        *reinterpret_cast<float2*>(reinterpret_cast<float*>(out) + oi) = make_float2(x0, x1);
    }
    if (lse != nullptr && t4 == 0) lse[row] = (m + log2f(l)) * 0.69314718055994531f;
  };
  store(plo, m_lo, l_lo, 0);
  store(phi, m_hi, l_hi, 1);
}

}  // namespace

cudaError_t launch_prefill(int32_t n_tokens, int32_t prefix_len, int32_t n_branches, const int32_t* branch_len,
                           int32_t h_q, int32_t h_kv, int32_t head_dim, float scale, int32_t out_bf16, const void* q,
                           const void* k, const void* v, void* out, float* lse, cudaStream_t s) {
  if (n_branches < 0 || n_branches > kMaxBranches) return cudaErrorInvalidValue;
  PrefillParams pp;
  pp.n_tokens = n_tokens;
  pp.prefix_len = prefix_len;
  pp.n_branches = n_branches;
  pp.h_q = h_q;
  pp.h_kv = h_kv;
  pp.group = h_q / h_kv;
  pp.scale_log2 = (float)((double)scale * 1.4426950408889634);
  pp.out_bf16 = out_bf16;
  pp.bstart[0] = prefix_len;
  for (int b = 0; b < n_branches; ++b) pp.bstart[b + 1] = pp.bstart[b] + branch_len[b];
  if (n_tokens == 0) return cudaSuccess;
  const dim3 grid((n_tokens + kTM - 1) / kTM, h_q);
  auto Q = static_cast<const __nv_bfloat16*>(q);
  auto K = static_cast<const __nv_bfloat16*>(k);
  auto V = static_cast<const __nv_bfloat16*>(v);
  if (head_dim == 128) {
    const size_t smem = (size_t)2 * 2 * kTN * (128 + 8) * 2;
    static bool configured = false;
    if (!configured) {
      cudaError_t e = cudaFuncSetAttribute(prefill_mma_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)smem);
      if (e != cudaSuccess) return e;
      configured = true;
    }
    prefill_mma_kernel<128><<<grid, kThreads, smem, s>>>(pp, Q, K, V, out, lse);
  } else if (head_dim == 64) {
    const size_t smem = (size_t)2 * 2 * kTN * (64 + 8) * 2;
    prefill_mma_kernel<64><<<grid, kThreads, smem, s>>>(pp, Q, K, V, out, lse);
  } else {
    return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace pad
