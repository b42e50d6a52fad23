// Grounding readout of the planning tokens (Sec. 3.3, and the paper's note on inference by
// similarity matching): each generated event token G^i is matched against the audio-visual
// prefix tokens after both went through the model's projection; the dot products of one
// time segment's tokens are summed into a segment score, and the segments whose score
// reaches a fraction of the event's best form its grounded interval.  Attention-guided
// aggregation (strategy (3) of Sec. 3.3) then pools the grounded tokens' hidden states with
// the last query token's attention weights and adds the result to the event embedding.
//
// The segment score is linear in the token features, so sum_t <g, f_t> = <g, sum_t f_t>:
// the prefix is read once, pooling each segment's projected features (ground_pool_kernel,
// HBM-bound; loads are issued four at a time per thread, since a latency-bound stream of
// single loads ran at a twentieth of the bandwidth), and scoring every event against the pooled rows is a small contraction over
// L2-resident data (ground_score_kernel).  The aggregation reads the hidden states once,
// pooling them per segment with the attention weights, and sums each event's segments
// (attn_seg_pool_kernel, attn_event_kernel).
#include <cuda_bf16.h>
#include <algorithm>
#include <cstdint>

#include "pad_internal.h"

namespace pad {
namespace {

constexpr int kThreads = 256;
constexpr int kMaxSegments = 1024;

struct Offsets {
  int32_t n;                       // segments
  int32_t off[kMaxSegments + 1];   // token ranges [off[s], off[s + 1])
};

// 16-byte streaming load, issued where it stands (asm volatile keeps a group of them ahead
// of their first use, so that they are in flight together).
__device__ __forceinline__ uint4 ld_stream(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

// Four such loads in one statement: all four are issued before any of them is used.
__device__ __forceinline__ void ld_stream4(uint4 (&v)[4], const void* p0, const void* p1, const void* p2,
                                           const void* p3) {
  asm volatile(
      "ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%16];\n"
      "ld.global.nc.L1::no_allocate.v4.u32 {%4, %5, %6, %7}, [%17];\n"
      "ld.global.nc.L1::no_allocate.v4.u32 {%8, %9, %10, %11}, [%18];\n"
      "ld.global.nc.L1::no_allocate.v4.u32 {%12, %13, %14, %15}, [%19];"
      : "=r"(v[0].x), "=r"(v[0].y), "=r"(v[0].z), "=r"(v[0].w), "=r"(v[1].x), "=r"(v[1].y), "=r"(v[1].z),
        "=r"(v[1].w), "=r"(v[2].x), "=r"(v[2].y), "=r"(v[2].z), "=r"(v[2].w), "=r"(v[3].x), "=r"(v[3].y),
        "=r"(v[3].z), "=r"(v[3].w)
      : "l"(p0), "l"(p1), "l"(p2), "l"(p3));
}

__device__ __forceinline__ void unpack8(const uint4 v, float* f) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const float2 t = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[j]));
    f[2 * j] = t.x;
    f[2 * j + 1] = t.y;
  }
}

// Grid (segment, slice of 4 * RP rows): the 256 threads cover the row's 16-byte chunks
// (CH = d / 8 of them) and RP = 256 / CH rows at a time, four rows per thread loaded
// together; the RP partial sums are added in shared memory and then into seg_sum (zeroed
// by the launcher) with atomics, so the slices of a segment add up in no fixed order.
constexpr int kPoolRowsPerThread = 16;
__global__ void __launch_bounds__(kThreads) ground_pool_kernel(const __grid_constant__ Offsets so,
                                                               const __nv_bfloat16* __restrict__ f, int d,
                                                               float* __restrict__ seg_sum) {
  extern __shared__ float red[];  // [RP][d]
  const int s = blockIdx.x;
  const int CH = d / 8, RP = kThreads / CH;
  const int c = threadIdx.x % CH, rg = threadIdx.x / CH;
  const int lo = so.off[s] + blockIdx.y * kPoolRowsPerThread * RP, hi = so.off[s + 1];
  if (lo >= hi) return;  // uniform over the CTA
  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  if (rg < RP) {
    const int t = lo + rg;
    if (t + (kPoolRowsPerThread - 1) * RP < hi) {
      // sixteen rows per thread, issued in groups of four
      uint4 v[4][4];
#pragma unroll
      for (int g = 0; g < 4; ++g) {
        const int tg = t + 4 * g * RP;
        ld_stream4(v[g], reinterpret_cast<const uint4*>(f + (size_t)tg * d) + c,
                   reinterpret_cast<const uint4*>(f + (size_t)(tg + RP) * d) + c,
                   reinterpret_cast<const uint4*>(f + (size_t)(tg + 2 * RP) * d) + c,
                   reinterpret_cast<const uint4*>(f + (size_t)(tg + 3 * RP) * d) + c);
      }
#pragma unroll
      for (int g = 0; g < 4; ++g)
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          float x[8];
          unpack8(v[g][u], x);
#pragma unroll
          for (int j = 0; j < 8; ++j) acc[j] += x[j];
        }
    } else {
      for (int u = 0; u < kPoolRowsPerThread && t + u * RP < hi; ++u) {
        float x[8];
        unpack8(__ldg(reinterpret_cast<const uint4*>(f + (size_t)(t + u * RP) * d) + c), x);
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[j] += x[j];
      }
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) red[rg * d + c * 8 + j] = acc[j];
  }
  __syncthreads();
  for (int i = threadIdx.x; i < d; i += kThreads) {
    float tot = 0.f;
    for (int r = 0; r < RP; ++r) tot += red[r * d + i];
    atomicAdd(seg_sum + (size_t)s * d + i, tot);
  }
}

// One CTA per event: scores against every pooled segment row, the best score, the salient
// set (score >= fraction * best when best > 0, else the first best segment alone) and the
// first and last salient segments.
__global__ void __launch_bounds__(kThreads) ground_score_kernel(const __nv_bfloat16* __restrict__ g, int S, int d,
                                                                const float* __restrict__ seg_sum, float frac,
                                                                float* __restrict__ scores,
                                                                uint8_t* __restrict__ salient,
                                                                int32_t* __restrict__ interval) {
  extern __shared__ float gs[];  // [d] the event's projected token, then [S] scores
  float* sc = gs + d;
  __shared__ float wbest[kThreads / 32];
  __shared__ int wlo[kThreads / 32], whi[kThreads / 32], warg[kThreads / 32];
  const int i = blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int c = threadIdx.x; c < d; c += kThreads) gs[c] = __bfloat162float(g[(size_t)i * d + c]);
  __syncthreads();
  // a warp per segment row (lanes over its float4 columns), eight rows in flight per warp
  float best = -__builtin_huge_valf();
  const int d4 = d / 4;
  for (int s0 = warp * 8; s0 < S; s0 += 8 * (kThreads / 32)) {
    float part[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    for (int c = lane; c < d4; c += 32) {
      float4 v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u)
        v[u] = s0 + u < S ? __ldg(reinterpret_cast<const float4*>(seg_sum + (size_t)(s0 + u) * d) + c)
                          : make_float4(0.f, 0.f, 0.f, 0.f);
      const float g0 = gs[4 * c], g1 = gs[4 * c + 1], g2 = gs[4 * c + 2], g3 = gs[4 * c + 3];
#pragma unroll
      for (int u = 0; u < 8; ++u) part[u] += (g0 * v[u].x + g1 * v[u].y) + (g2 * v[u].z + g3 * v[u].w);
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      float v = part[u];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
      if (s0 + u < S) {
        if (lane == 0) {
          sc[s0 + u] = v;
          scores[(size_t)i * S + s0 + u] = v;
        }
        best = fmaxf(best, v);
      }
    }
  }
  __syncthreads();
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) best = fmaxf(best, __shfl_xor_sync(0xffffffffu, best, o));
  if (lane == 0) wbest[warp] = best;
  __syncthreads();
  best = wbest[0];
  for (int w = 1; w < kThreads / 32; ++w) best = fmaxf(best, wbest[w]);
  // the first best segment (used alone when no score is positive)
  int arg = S;
  for (int s = threadIdx.x; s < S; s += kThreads)
    if (sc[s] == best) arg = min(arg, s);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) arg = min(arg, __shfl_xor_sync(0xffffffffu, arg, o));
  if (lane == 0) warg[warp] = arg;
  __syncthreads();
  arg = warg[0];
  for (int w = 1; w < kThreads / 32; ++w) arg = min(arg, warg[w]);
  const float cut = frac * best;
  int lo = S, hi = -1;
  for (int s = threadIdx.x; s < S; s += kThreads) {
    const bool on = best > 0.f ? sc[s] >= cut : s == arg;
    salient[(size_t)i * S + s] = on ? 1 : 0;
    if (on) {
      lo = min(lo, s);
      hi = max(hi, s);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    lo = min(lo, __shfl_xor_sync(0xffffffffu, lo, o));
    hi = max(hi, __shfl_xor_sync(0xffffffffu, hi, o));
  }
  if (lane == 0) {
    wlo[warp] = lo;
    whi[warp] = hi;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int w = 1; w < kThreads / 32; ++w) {
      lo = min(lo, wlo[w]);
      hi = max(hi, whi[w]);
    }
    lo = min(lo, wlo[0]);
    hi = max(hi, whi[0]);
    interval[2 * i] = lo;
    interval[2 * i + 1] = hi;
  }
}

// Attention-guided aggregation.  The weights attn[t] belong to the tokens, not to the
// events, so an event's weighted sum over its grounded segments lo..hi is the sum of the
// segments' own weighted sums: the hidden states are read once (attn_seg_pool_kernel,
// HBM-bound), and every event then adds up its segments' rows, which stay in L2
// (attn_event_kernel).  For balance the token axis is cut into pieces of at most
// kAggPiece tokens, each inside one segment (segment s owns pieces pbeg[s] .. pbeg[s+1]-1),
// and the pooled rows are per piece: W[p] = sum_{t in p} attn[t] x[t], A[p] = sum_{t in p}
// attn[t].  Every element is written once and summed in a fixed order, so the results are
// the same from run to run.
constexpr int kAggCols = 256;
constexpr int kAggPiece = 256;
constexpr int kAggGroups = kThreads / 32;

struct Pieces {
  int32_t n;                          // segments
  int32_t off[kMaxSegments + 1];      // token ranges of the segments
  int32_t pbeg[kMaxSegments + 1];     // first piece of each segment; pbeg[n] = pieces
};

// attn_seg_pool_kernel: grid (piece, slice of kAggCols columns).  Eight row groups of 32
// threads; a thread owns one 16-byte piece (8 columns) of every eighth row and keeps eight
// rows' loads in flight; the row groups' sums are added in shared memory, in order.
__global__ void __launch_bounds__(kThreads) attn_seg_pool_kernel(const __grid_constant__ Pieces pm,
                                                                 const __nv_bfloat16* __restrict__ x, int d,
                                                                 const float* __restrict__ attn,
                                                                 float* __restrict__ wsum, float* __restrict__ asum) {
  __shared__ float red[kAggGroups][kAggCols];
  __shared__ float ared[kAggGroups];
  const int pc = blockIdx.x;
  int sl = 0, sh = pm.n - 1;  // the segment owning piece pc: the last s with pbeg[s] <= pc
  while (sl < sh) {
    const int mid = (sl + sh + 1) >> 1;
    if (pm.pbeg[mid] <= pc)
      sl = mid;
    else
      sh = mid - 1;
  }
  const int lo = pm.off[sl] + (pc - pm.pbeg[sl]) * kAggPiece, hi = min(pm.off[sl + 1], lo + kAggPiece);
  const int lane = threadIdx.x & 31, rg = threadIdx.x >> 5;
  const int c = blockIdx.y * (kAggCols / 8) + lane;  // 16-byte piece of the row
  const bool cin = c < d / 8;
  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  float wacc = 0.f;
  const uint4* xc = reinterpret_cast<const uint4*>(x) + (cin ? c : 0);
  const size_t rs = (size_t)d / 8;  // row stride in pieces
  int t = lo + rg;
  for (; t + 7 * kAggGroups < hi; t += 8 * kAggGroups) {
    uint4 v[2][4];
    ld_stream4(v[0], xc + (size_t)t * rs, xc + (size_t)(t + kAggGroups) * rs, xc + (size_t)(t + 2 * kAggGroups) * rs,
               xc + (size_t)(t + 3 * kAggGroups) * rs);
    ld_stream4(v[1], xc + (size_t)(t + 4 * kAggGroups) * rs, xc + (size_t)(t + 5 * kAggGroups) * rs,
               xc + (size_t)(t + 6 * kAggGroups) * rs, xc + (size_t)(t + 7 * kAggGroups) * rs);
    float w[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) w[u] = __ldg(attn + t + u * kAggGroups);
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      float f[8];
      unpack8(v[u >> 2][u & 3], f);
#pragma unroll
      for (int j = 0; j < 8; ++j) acc[j] = fmaf(w[u], f[j], acc[j]);
      wacc += w[u];
    }
  }
  for (; t < hi; t += kAggGroups) {
    const float w0 = __ldg(attn + t);
    float f[8];
    unpack8(__ldg(xc + (size_t)t * rs), f);
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[j] = fmaf(w0, f[j], acc[j]);
    wacc += w0;
  }
#pragma unroll
  for (int j = 0; j < 8; ++j) red[rg][lane * 8 + j] = acc[j];
  if (lane == 0) ared[rg] = wacc;  // (every lane of the group summed the same weights)
  __syncthreads();
  const int col = blockIdx.y * kAggCols + threadIdx.x;
  if (col < d) {
    float tot = 0.f;
#pragma unroll
    for (int r = 0; r < kAggGroups; ++r) tot += red[r][threadIdx.x];
    wsum[(size_t)pc * d + col] = tot;
  }
  if (blockIdx.y == 0 && threadIdx.x == 0) {
    float a = 0.f;
    for (int r = 0; r < kAggGroups; ++r) a += ared[r];
    asum[pc] = a;
  }
}

// attn_event_kernel: grid (event, slice of kAggCols columns).  The pieces of the event's
// interval (lo, hi), clamped to the segments, are spread over the eight warps (warp w takes
// every eighth piece from the first); a lane adds 8 columns; the warps' sums are added in
// shared memory, in order, and out = g_emb + sum W / sum A (g_emb alone when sum A is 0).
__global__ void __launch_bounds__(kThreads) attn_event_kernel(const __grid_constant__ Pieces pm, int d,
                                                              const int32_t* __restrict__ interval,
                                                              const float* __restrict__ wsum,
                                                              const float* __restrict__ asum,
                                                              const __nv_bfloat16* __restrict__ g_emb,
                                                              float* __restrict__ out) {
  __shared__ float red[kAggGroups][kAggCols];
  __shared__ float ared[kAggGroups];
  const int i = blockIdx.x, S = pm.n;
  const int s_lo = min(max(interval[2 * i], 0), S - 1), s_hi = min(max(interval[2 * i + 1], s_lo), S - 1);
  const int p0 = pm.pbeg[s_lo], p1 = pm.pbeg[s_hi + 1];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int c8 = blockIdx.y * kAggCols + lane * 8;  // first of this lane's 8 columns
  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  float a = 0.f;
  if (c8 < d) {
    for (int pc = p0 + w; pc < p1; pc += kAggGroups) {
      const float4* src = reinterpret_cast<const float4*>(wsum + (size_t)pc * d + c8);
      const float4 u0 = __ldg(src), u1 = __ldg(src + 1);
      acc[0] += u0.x;
      acc[1] += u0.y;
      acc[2] += u0.z;
      acc[3] += u0.w;
      acc[4] += u1.x;
      acc[5] += u1.y;
      acc[6] += u1.z;
      acc[7] += u1.w;
      a += __ldg(asum + pc);
    }
  }
#pragma unroll
  for (int j = 0; j < 8; ++j) red[w][lane * 8 + j] = acc[j];
  if (lane == 0) ared[w] = a;
  __syncthreads();
  const int col = blockIdx.y * kAggCols + threadIdx.x;
  if (col < d) {
    float num = 0.f, den = 0.f;
#pragma unroll
    for (int r = 0; r < kAggGroups; ++r) {
      num += red[r][threadIdx.x];
      den += ared[r];
    }
    const float base = __bfloat162float(g_emb[(size_t)i * d + col]);
    out[(size_t)i * d + col] = den > 0.f ? base + num / den : base;
  }
}

bool fill_offsets(Offsets& so, const int32_t* offsets, int32_t n_segments, int64_t n_tokens) {
  if (n_segments < 1 || n_segments > kMaxSegments || !offsets) return false;
  so.n = n_segments;
  for (int s = 0; s <= n_segments; ++s) {
    if (offsets[s] < 0 || offsets[s] > n_tokens || (s > 0 && offsets[s] < offsets[s - 1])) return false;
    so.off[s] = offsets[s];
  }
  return true;
}

}  // namespace

cudaError_t launch_ground_pool(const void* f_proj, int64_t n_tokens, int32_t d, const int32_t* offsets,
                               int32_t n_segments, float* seg_sum, cudaStream_t s) {
  Offsets so;
  if (!fill_offsets(so, offsets, n_segments, n_tokens)) return cudaErrorInvalidValue;
  const int CH = d / 8, RP = kThreads / CH;
  int longest = 0;
  for (int i = 0; i < n_segments; ++i) longest = std::max(longest, so.off[i + 1] - so.off[i]);
  const int slices = std::max(1, (longest + kPoolRowsPerThread * RP - 1) / (kPoolRowsPerThread * RP));
  if (slices > 65535) return cudaErrorInvalidValue;
  cudaError_t e = cudaMemsetAsync(seg_sum, 0, (size_t)n_segments * d * sizeof(float), s);
  if (e != cudaSuccess) return e;
  ground_pool_kernel<<<dim3(n_segments, slices), kThreads, (size_t)RP * d * sizeof(float), s>>>(
      so, static_cast<const __nv_bfloat16*>(f_proj), d, seg_sum);
  return cudaGetLastError();
}

cudaError_t launch_ground_score(const void* g_proj, int32_t n_events, const float* seg_sum, int32_t n_segments,
                                int32_t d, float frac, float* scores, uint8_t* salient, int32_t* interval,
                                cudaStream_t s) {
  if (n_events == 0) return cudaSuccess;
  const size_t smem = (size_t)(d + n_segments) * sizeof(float);
  ground_score_kernel<<<n_events, kThreads, smem, s>>>(static_cast<const __nv_bfloat16*>(g_proj), n_segments, d,
                                                       seg_sum, frac, scores, salient, interval);
  return cudaGetLastError();
}

size_t attn_aggregate_ws_floats(int64_t n_tokens, int32_t n_segments, int32_t d) {
  return ((size_t)n_segments + (size_t)(n_tokens + kAggPiece - 1) / kAggPiece) * ((size_t)d + 1);
}

cudaError_t launch_attn_aggregate(const void* x, int64_t n_tokens, int32_t d, const float* attn,
                                  const int32_t* offsets, int32_t n_segments, const int32_t* interval,
                                  int32_t n_events, const void* g_emb, float* seg_ws, float* out, cudaStream_t s) {
  Offsets so;
  if (!fill_offsets(so, offsets, n_segments, n_tokens)) return cudaErrorInvalidValue;
  if (n_events == 0) return cudaSuccess;
  Pieces pm;
  pm.n = n_segments;
  pm.pbeg[0] = 0;
  for (int i = 0; i < n_segments; ++i) {
    pm.off[i] = so.off[i];
    pm.pbeg[i + 1] = pm.pbeg[i] + (so.off[i + 1] - so.off[i] + kAggPiece - 1) / kAggPiece;
  }
  pm.off[n_segments] = so.off[n_segments];
  const int pieces = pm.pbeg[n_segments];
  const int slices = (d + kAggCols - 1) / kAggCols;
  if (slices > 65535) return cudaErrorInvalidValue;
  // (pieces <= n_segments + n_tokens / kAggPiece: within attn_aggregate_ws_floats)
  float* wsum = seg_ws;
  float* asum = seg_ws + (size_t)std::max(pieces, 1) * d;
  if (pieces > 0) {
    attn_seg_pool_kernel<<<dim3(pieces, slices), kThreads, 0, s>>>(pm, static_cast<const __nv_bfloat16*>(x), d, attn,
                                                                   wsum, asum);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  attn_event_kernel<<<dim3(n_events, slices), kThreads, 0, s>>>(pm, d, interval, wsum, asum,
                                                                 static_cast<const __nv_bfloat16*>(g_emb), out);
  return cudaGetLastError();
}

}  // namespace pad
