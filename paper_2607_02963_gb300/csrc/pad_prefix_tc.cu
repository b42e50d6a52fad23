// a3 on the 5th-generation tensor cores: split-KV flash-decode over the shared
// prefix (the part of the event-factorized mask of Sec. 3.4 that every branch
// of a video sees: the multimodal prefix P and all planning tokens G^1..G^K, S).
//
// One CTA per (work item = video, kv-head, prefix split; group of <= 128 query
// rows).  The R = E_b * G query rows of the video's events that read this
// kv-head form the M dimension of the MMA, so each K/V tile brought from HBM
// serves every event and every GQA head of the group at once; the row groups of
// one item are adjacent CTAs that run together and share the tiles through L2.
//
//   warp 0      TMA producer of K tiles (128 tokens: two 64-column halves, 128-byte
//               swizzle) into a 3-stage ring; a stage is refilled once the S of
//               the tile it held has completed
//   warp 1      S issuer (one thread): S = Q K^T into one of three TMEM S buffers,
//               up to three tiles ahead of the softmax
//   warp 2      TMEM allocator (512 columns) and deallocator; its lane 0 issues
//               O += P V with P read back from TMEM
//   warp 3      TMA producer of V tiles (refilled once the P.V of the tile completed)
//   warps 4-11  softmax: two warps per 32-row lane quarter.  Decode: each warp takes 16
//               of the quarter's rows and all 128 columns of a tile (two rows per
//               thread, a row shared by a quad of lanes), so the warps never meet.
//               Whole-sequence prefill: each takes 64 of the columns for one row per
//               thread, and the two meet once per tile to combine their partial row
//               maxima (an mbarrier, so the wait is bounded).  Online max and sum in
//               base 2, P written as packed bf16 over the S columns already read, lazy
//               rescaling of O (only when a row maximum grows by more than 2^8)
//
// Every MMA has N = 128 (S: 128 tokens; P.V: 128 head-dim columns), the size at
// which one tcgen05.mma carries as much tensor work as it costs to issue.
// TMEM columns: S[b] at 128*b (b = 0, 1, 2), O at 384.  Output: the partial
// softmax state (m, l, O) of every row for this split, merged with the other
// splits and the branch by the branch/merge kernel, or, when the plan fuses them
// (every (event, kv-head) task has a CTA of its own and the grid is one wave), by
// the softmax warps of this kernel after their split: they publish the split on a
// counter, then run one task's branch pass, wait for the counters of the task's rows
// and merge (a4 + a5 as in the standalone kernel, same code).
//
// Barrier phases: a thread waits for completion #c of a barrier by its parity, which is
// only sound while completion #c+1 cannot yet have happened.  Every barrier here is
// therefore per slot (stage, S buffer, or tile parity) so that its next completion
// depends on progress of the waiting thread itself.
//
// Every mbarrier wait is bounded (about one second of %globaltimer); a wait
// that runs out records PAD_ERR_DEVICE_TIMEOUT in the status word, raises a
// CTA-wide abort flag, lets the producers and the MMA issuer drain what they
// already started, frees TMEM and returns.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <algorithm>
#include <cstddef>
#include <cstdint>
#include <cstring>
#include <mutex>

#include "pad_branch_merge.cuh"
#include "pad_internal.h"
#include "pad_tc_common.cuh"

namespace pad {

namespace {

using namespace tc;

constexpr int kD = 128;
constexpr int kBN = 128;       // prefix tokens per K/V tile
constexpr int kStages = 3;
constexpr int kSBuf = 3;       // S buffers in TMEM
constexpr int kThreads = 384;
constexpr uint32_t kHalfBytes = kBN * 128;         // 128 tokens x 64 bf16 = 16 KB
constexpr uint32_t kTileBytes = 2 * kHalfBytes;    // one K (or V) tile: 32 KB
constexpr uint32_t kQHalfBytes = 128 * 128;        // 128 rows x 64 bf16 = 16 KB
constexpr uint32_t kQTileBytes = 2 * kQHalfBytes;  // Q of one 128-row group: 32 KB
constexpr uint32_t kOffQ = 0;
constexpr uint32_t kOffK = kOffQ + kQTileBytes;
constexpr uint32_t kOffV = kOffK + kStages * kTileBytes;
constexpr uint32_t kOffBar = kOffV + kStages * kTileBytes;
constexpr uint32_t kOffX = kOffBar + 256;               // prefill: partial row maxima [2][2][128] fp32
constexpr uint32_t kSmemBytes = kOffX + 2 * 2 * 128 * 4;
constexpr int kOStage = kD + 4;                       // fp32 row stride of the O staging rows
static_assert((128 * kOStage + 128) * 4 <= kStages * kTileBytes, "O staging (and 1 / l) fits the K stages");
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColO = 384;
constexpr float kLazyRescale = 8.0f;                  // log2 units
static_assert(kSmemBytes <= 232448, "fits the 227 KB opt-in shared memory");

struct TcBars {
  uint64_t kfull[kStages];
  uint64_t vfull[kStages];
  uint64_t pvfree[kStages];   // P.V of the tile in this stage / S buffer has completed
  uint64_t sfull[kSBuf];      // S of the tile in this buffer has completed (also frees its K stage)
  uint64_t pfull[kSBuf];      // P of the tile in this buffer is written (8 warp arrivals)
  uint64_t drain_s;           // every S MMA has completed (S issuer)
  uint64_t drain_pv;          // every P.V MMA has completed (P.V issuer)
  uint64_t qready;            // Q staged in shared memory (8 warp arrivals)
  uint64_t tdone;             // the softmax warps are done with TMEM (8 warp arrivals)
  uint64_t xchg[4];           // prefill: the two softmax warps of a lane quarter met (64 arrivals)
  uint64_t gen;               // the plan's generation, for the status word
  uint32_t tmem_base;
  int32_t abort;
};
static_assert(sizeof(TcBars) <= 256, "barrier block fits its slot");

constexpr uint32_t kIdescS = make_idesc(128, kBN, false);   // S = Q K^T: B = K tile, K-major
constexpr uint32_t kIdescPV = make_idesc(128, kD, true);    // O += P V: B = V tile, N(=d)-major

// The prefill path splits a 128-row group by columns: the two warps of a lane quarter take
// 64 columns each of its 32 rows (one row per thread) and meet on every tile to share their
// row maxima; one causal mask per thread keeps it below the register limit, where two rows'
// masks per thread spilled.
// Visible columns of a warp's 64 (used on the MASK path only): the set bits of `keep`.
struct HalfBits {
  uint64_t keep;
  __device__ bool vis(int c) const { return (keep >> c) & 1ull; }
};
// Maximum of the raw scores of one softmax warp's 64 columns (eight chains of three-input
// max); with MASK, columns the row does not see are left out.
template <bool MASK, class Cols>
__device__ __forceinline__ float half_row_max(const uint32_t (&sr)[2][32], Cols cols) {
  float mxa[8];
#pragma unroll
  for (int u = 0; u < 8; ++u) mxa[u] = -__builtin_huge_valf();
#pragma unroll
  for (int c = 0; c < 2; ++c)
#pragma unroll
    for (int i = 0; i < 32; i += 2) {
      float a = __uint_as_float(sr[c][i]), b = __uint_as_float(sr[c][i + 1]);
      if (MASK) {
        if (!cols.vis(32 * c + i)) a = -__builtin_huge_valf();
        if (!cols.vis(32 * c + i + 1)) b = -__builtin_huge_valf();
      }
      const int u = (16 * c + i / 2) & 7;
      mxa[u] = max3f(mxa[u], a, b);
    }
  return fmaxf(max3f(mxa[0], mxa[1], mxa[2]), max3f(max3f(mxa[3], mxa[4], mxa[5]), mxa[6], mxa[7]));
}

// P = 2^(s * scale_log2 - m) for one softmax warp's 64 columns, written as packed bf16
// over the S columns already read; returns the fp32 sum of the P values.
template <bool MASK, class Cols>
__device__ __forceinline__ float half_row_exp(const uint32_t (&sr)[2][32], Cols cols, float sl2,
                                              float m, uint32_t taddr_p);

template <bool MASK, class Cols>
__device__ __forceinline__ float half_row_exp(const uint32_t (&sr)[2][32], Cols cols, float sl2,
                                              float m, uint32_t taddr_p) {
  const uint64_t sc2 = f2pack(sl2, sl2), nm2 = f2pack(-m, -m);
  uint64_t lacc[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
  for (int c = 0; c < 2; ++c) {
    uint32_t pk[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const int col = 32 * c + 2 * i;
      const uint64_t x =
          ffma2(f2pack(__uint_as_float(sr[c][2 * i]), __uint_as_float(sr[c][2 * i + 1])), sc2, nm2);
      float p0 = ex2(f2lo(x)), p1 = ex2(f2hi(x));
      if (MASK) {
        if (!cols.vis(col)) p0 = 0.f;
        if (!cols.vis(col + 1)) p1 = 0.f;
      }
      lacc[i & 3] = fadd2(lacc[i & 3], f2pack(p0, p1));
      pk[i] = pack_bf16(p0, p1);
    }
    // P of tokens 32c .. 32c+31 of this half, two per column
    tmem_st16(taddr_p + 16 * c, pk);
  }
  const uint64_t ls = fadd2(fadd2(lacc[0], lacc[1]), fadd2(lacc[2], lacc[3]));
  return f2lo(ls) + f2hi(ls);
}


// The softmax warps split a 128-row group by rows: warp w of lane quarter q takes the 16
// rows 32q + 16h .. +15 (h = (w-4)/4) and every column of a tile, through the 16-lane TMEM
// shapes, so no row is shared by two warps and they never have to meet.  Thread t holds rows
// a = t/4 and a + 8 of the warp's 16 and, in each 8-column chunk, columns 2(t%4) and
// 2(t%4) + 1: s[x][4k..4k+3] = (a, c), (a, c+1), (a+8, c), (a+8, c+1) with
// c = 64x + 8k + 2(t%4).  A row's maximum and sum are shared by the four threads of its
// quad (lanes 4(t/4) .. +3).
// Visible columns of one row: the first `valid`, or the set bits of a 128-column mask.
struct ColsValid {
  int valid;
  __device__ bool vis(int c) const { return c < valid; }
};
struct ColsBits {
  uint64_t lo, hi;  // columns 0-63, 64-127
  __device__ bool vis(int c) const { return ((c < 64 ? lo >> c : hi >> (c - 64)) & 1ull) != 0; }
};
__device__ __forceinline__ float quad_max(float v) {
  v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 1));
  return fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 2));
}
__device__ __forceinline__ float quad_sum(float v) {
  v += __shfl_xor_sync(0xffffffffu, v, 1);
  return v + __shfl_xor_sync(0xffffffffu, v, 2);
}

// Maxima of the raw scores of this thread's two rows over all 128 columns (with MASK,
// columns a row does not see are left out), reduced over the quad.
template <bool MASK, class CA, class CB>
__device__ __forceinline__ void rows_max(const uint32_t (&s)[2][32], int cq, CA ca, CB cb, float& ma, float& mb) {
  float xa[4], xb[4];
#pragma unroll
  for (int u = 0; u < 4; ++u) xa[u] = xb[u] = -__builtin_huge_valf();
#pragma unroll
  for (int x = 0; x < 2; ++x)
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const int c = 64 * x + 8 * k + cq;
      float a0 = __uint_as_float(s[x][4 * k]), a1 = __uint_as_float(s[x][4 * k + 1]);
      float b0 = __uint_as_float(s[x][4 * k + 2]), b1 = __uint_as_float(s[x][4 * k + 3]);
      if (MASK) {
        if (!ca.vis(c)) a0 = -__builtin_huge_valf();
        if (!ca.vis(c + 1)) a1 = -__builtin_huge_valf();
        if (!cb.vis(c)) b0 = -__builtin_huge_valf();
        if (!cb.vis(c + 1)) b1 = -__builtin_huge_valf();
      }
      xa[k & 3] = max3f(xa[k & 3], a0, a1);
      xb[k & 3] = max3f(xb[k & 3], b0, b1);
    }
  ma = quad_max(fmaxf(fmaxf(xa[0], xa[1]), fmaxf(xa[2], xa[3])));
  mb = quad_max(fmaxf(fmaxf(xb[0], xb[1]), fmaxf(xb[2], xb[3])));
}

// P = 2^(s * scale_log2 - m) of this thread's two rows, written as packed bf16 (two tokens
// per column: column 4k + t%4 of chunk k holds tokens 8k + 2(t%4) and + 1, the layout the
// P.V MMA reads) to the 64 TMEM columns at taddr_p; adds this thread's share of each row's
// sum of P to la / lb.
template <bool MASK, class CA, class CB>
__device__ __forceinline__ void rows_exp(const uint32_t (&s)[2][32], int cq, CA ca, CB cb, float sl2, float ma,
                                         float mb, uint32_t taddr_p, float& la, float& lb) {
  const uint64_t sc2 = f2pack(sl2, sl2), na = f2pack(-ma, -ma), nb = f2pack(-mb, -mb);
  uint64_t acc_a[2] = {0ull, 0ull}, acc_b[2] = {0ull, 0ull};
#pragma unroll
  for (int x = 0; x < 2; ++x) {
    uint32_t pk[16];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const int c = 64 * x + 8 * k + cq;
      const uint64_t ya =
          ffma2(f2pack(__uint_as_float(s[x][4 * k]), __uint_as_float(s[x][4 * k + 1])), sc2, na);
      const uint64_t yb =
          ffma2(f2pack(__uint_as_float(s[x][4 * k + 2]), __uint_as_float(s[x][4 * k + 3])), sc2, nb);
      float a0 = ex2(f2lo(ya)), a1 = ex2(f2hi(ya)), b0 = ex2(f2lo(yb)), b1 = ex2(f2hi(yb));
      if (MASK) {
        if (!ca.vis(c)) a0 = 0.f;
        if (!ca.vis(c + 1)) a1 = 0.f;
        if (!cb.vis(c)) b0 = 0.f;
        if (!cb.vis(c + 1)) b1 = 0.f;
      }
      acc_a[k & 1] = fadd2(acc_a[k & 1], f2pack(a0, a1));
      acc_b[k & 1] = fadd2(acc_b[k & 1], f2pack(b0, b1));
      pk[2 * k] = pack_bf16(a0, a1);
      pk[2 * k + 1] = pack_bf16(b0, b1);
    }
    // P columns 32x + 4k + t%4 (tokens 64x + 8k + 2(t%4), + 1)
    tmem_st16x128_x8(taddr_p + 32 * x, pk);
  }
  const uint64_t sa = fadd2(acc_a[0], acc_a[1]), sb = fadd2(acc_b[0], acc_b[1]);
  la += f2lo(sa) + f2hi(sa);
  lb += f2lo(sb) + f2hi(sb);
}

// Bounded wait of this kernel: gives up on the CTA's abort flag or after the time limit.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, TcBars* bars,
                                          PadDevHeader* hdr, int where) {
  return mbar_wait_b(bar, parity, &bars->abort, bars->gen, hdr, where);
}


// Split counters of the fused tail, one per (video, kv-head, 128-row group): bits 15-0
// count the video's splits that have written their partial rows, bits 31-16 the tasks
// that have taken them.  The append kernel of the step zeroes them; the last task to
// take a counter zeroes it again for a launch of the same plan without an append.
__device__ __forceinline__ unsigned ld_acquire_u32(const unsigned* a) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(a) : "memory");
  return v;
}
// Thread `leader` waits (bounded) until every split of video `vd` has published the rows
// [r0, r0 + G) of kv-head `kvh`, then takes them; the result is the same for all 256
// threads of the softmax group.
__device__ __forceinline__ bool tail_partials_ready(const KParams& p, const PadVideoDesc& vd, int kvh,
                                                    int r0, bool leader) {
  bool good = true;
  if (leader) {
    const int G = p.group;
    const int gb = (vd.n_events * G + 127) >> 7;
    const int g0 = r0 >> 7, g1 = (r0 + G - 1) >> 7;
    unsigned* base = p.counters + vd.cnt_base + (size_t)kvh * gb;
    const unsigned long long t0 = globaltimer();
    for (int g = g0; g <= g1 && good; ++g) {
      while ((int)(ld_acquire_u32(base + g) & 0xffffu) != vd.n_splits) {
        // give up at once if this plan's kernels already recorded an error (a split that
        // failed never publishes), else after the usual bound
        const unsigned long long hw = *reinterpret_cast<volatile unsigned long long*>(&p.header->word);
        if (((hw >> 8) == p.gen && (hw & 0xffull) != 0) || globaltimer() - t0 > kWaitNs) {
          pad_set_error(p.header, p.gen, PAD_ERR_DEVICE_TIMEOUT, (int)blockIdx.x, g, 20);
          good = false;
          break;
        }
        __nanosleep(64);
      }
    }
    if (good) {
      for (int g = g0; g <= g1; ++g) {
        const int lo = (g << 7) / G, hi = min(vd.n_events - 1, ((g << 7) + 127) / G);
        const unsigned old = atomicAdd(base + g, 1u << 16);
        if ((int)(old >> 16) + 1 == hi - lo + 1) atomicExch(base + g, 0u);
      }
    }
  }
  return bm::SyncNamed{1}.all(good);
}

// Whole-sequence prefill (PREFILL): branch start of token p >= pf_S, from the branch
// offsets carried in the parameters.
__device__ __forceinline__ int pf_branch_start(const KParams& p, int t) {
  const int32_t* bs = reinterpret_cast<const int32_t*>(p.img);
  int lo = 0, hi = p.pf_nb - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (bs[mid] <= t) lo = mid; else hi = mid - 1;
  }
  return bs[lo];
}
// Bits c of [0, 64) with lo <= c < hi (clamped).
__device__ __forceinline__ uint64_t range_bits(int lo, int hi) {
  lo = max(lo, 0);
  hi = min(hi, 64);
  if (lo >= hi) return 0ull;
  const uint64_t up = hi >= 64 ? ~0ull : ((1ull << hi) - 1ull);
  return up & ~((1ull << lo) - 1ull);
}

template <bool ROPE, bool GSELF, bool PREFILL>
__global__ void __launch_bounds__(kThreads, 1)
    prefix_tc_kernel(const __grid_constant__ KParams p, const __nv_bfloat16* __restrict__ q, const int n_groups,
                     const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                     const __nv_bfloat16* __restrict__ kpool, const __nv_bfloat16* __restrict__ vpool,
                     void* __restrict__ out, float* __restrict__ lse) {
  extern __shared__ __align__(1024) uint8_t smem[];
  const uint32_t sbase = smem_u32(smem);
  if (sbase & 1023u) {  // the 128-byte swizzle atoms need 1024-byte alignment (never expected)
    if (threadIdx.x == 0) pad_set_error(p.header, p.gen, PAD_ERR_UNSUPPORTED, (int)blockIdx.x, (int)sbase, 0);
    return;
  }
  TcBars* bars = reinterpret_cast<TcBars*>(smem + kOffBar);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // One-call step (k_new set): this is the step's first kernel, launched so that it may
  // start while the grid before it (the previous step, or the caller's own kernel that
  // wrote q) finishes.  Barrier set-up and TMEM allocation overlap that grid; every thread
  // that touches global memory waits for it first (the Q loads, the first TMA issue),
  // and the block barrier after them orders everything else, including the release of
  // the grid behind this one.
  const bool one_call = p.k_new != nullptr;

  // the CTA's work item and 128-row group: from the plan's CTA list, or the dense grid
  int item, group;
  if (p.cta_map) {
    const int v = plan_tasks(p)[blockIdx.x];
    item = v >> 6;
    group = v & 63;
  } else {
    item = blockIdx.x / n_groups;
    group = blockIdx.x - item * n_groups;
  }
  PadWorkItem it;
  // PREFILL: the CTA's query tokens [it.first_event, +n_events) of kv-head it.kvh (query
  // tiles in descending order, so that the longest key ranges start first) see the keys
  // [0, pf_a_end) of the prefix and [pf_b_lo, pf_b_end) of the branches
  int pf_a_tiles = 0, pf_b_lo = 0, pf_a_end = 0, pf_last = 0;
  if (PREFILL) {
    const int n_qt = (p.pf_N + p.pf_tpc - 1) / p.pf_tpc;
    const int qt = n_qt - 1 - (int)blockIdx.x / p.h_kv;
    it.first_event = qt * p.pf_tpc;
    it.n_events = min(p.pf_tpc, p.pf_N - it.first_event);
    it.kvh = (int16_t)(blockIdx.x % p.h_kv);
    it.split = 0;
    it.tok0 = 0;
    it.tok_begin = 0;
    it.part_row0 = 0;
    const int last = it.first_event + it.n_events - 1;
    const int a_end = min(p.pf_S, last + 1);
    pf_a_end = a_end;
    pf_last = last;
    pf_a_tiles = (a_end + kBN - 1) / kBN;
    int b_tiles = 0;
    if (last >= p.pf_S) {
      pf_b_lo = pf_branch_start(p, max(it.first_event, p.pf_S));
      b_tiles = (last + 1 - pf_b_lo + kBN - 1) / kBN;
    }
    it.tok_end = (pf_a_tiles + b_tiles) * kBN;  // tile count; columns are masked per tile
  } else {
    it = plan_items(p)[item];
  }
  const int R = it.n_events * p.group;
  const int row0 = group * 128;
  if (row0 >= R) return;  // uniform over the CTA, before any barrier or allocation
  const int ntok = it.tok_end - it.tok_begin;
  const int n_tiles = (ntok + kBN - 1) / kBN;
  const int kvh = it.kvh;
  const int tok0 = (int)it.tok0;
  // first token of K/V tile t
  auto tile_tok = [&](int t) -> int {
    if (PREFILL) return t < pf_a_tiles ? t * kBN : pf_b_lo + (t - pf_a_tiles) * kBN;
    return tok0 + t * kBN;
  };

  // The softmax warps load their Q rows now, so that the loads overlap barrier set-up
  // and TMEM allocation; they are stored to shared memory after the block barrier.
  // Lane `lane` of warp w holds row 32*(w&3) + (lane+32i)/8, 16-byte chunk (lane+32i)%8
  // of head-dim half (w-4)/4.  Rows past R are zero.
  uint4 qv[8];
  if (warp >= 4) {
    if (one_call) asm volatile("griddepcontrol.wait;" ::: "memory");
    const int lane_base = 32 * (warp & 3), half = (warp - 4) >> 2;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int idx = lane + 32 * i;
      const int qrow = row0 + lane_base + (idx >> 3);
      qv[i] = make_uint4(0u, 0u, 0u, 0u);
      if (qrow < R) {
        const int el = qrow / p.group;
        const int gh = qrow - el * p.group;
        const __nv_bfloat16* qr = q + ((size_t)(it.first_event + el) * p.h_q + kvh * p.group + gh) * kD;
        const int d0 = half * 64 + (idx & 7) * 8;
        qv[i] = __ldg(reinterpret_cast<const uint4*>(qr + d0));
      }
    }
  }

  if (threadIdx.x == 0) {
    // The first K and V tile go out first (their barriers initialised, then the loads),
    // before the other barriers, TMEM allocation and the block barrier; the producer warps
    // issue the rest once that K tile has landed, so that every CTA's first tile is not
    // queued in DRAM behind the later tiles of all the others.  The prefix K/V is written by
    // no grid of the library's own that may run ahead of this one (and, by the call's
    // contract, by no grid that releases its dependents before its writes), so that tile is
    // requested even before the wait for the grid ahead; nothing else is.
    mbar_init(&bars->kfull[0], 1);
    mbar_init(&bars->vfull[0], 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmK)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmV)) : "memory");
    if (n_tiles > 0) {
      mbar_expect_tx(&bars->kfull[0], kTileBytes);
      tma_load_3d(sbase + kOffK, &tmK, 0, kvh, tile_tok(0), &bars->kfull[0]);
      tma_load_3d(sbase + kOffK + kHalfBytes, &tmK, 64, kvh, tile_tok(0), &bars->kfull[0]);
      mbar_expect_tx(&bars->vfull[0], kTileBytes);
      tma_load_3d(sbase + kOffV, &tmV, 0, kvh, tile_tok(0), &bars->vfull[0]);
      tma_load_3d(sbase + kOffV + kHalfBytes, &tmV, 64, kvh, tile_tok(0), &bars->vfull[0]);
    }
    if (one_call) asm volatile("griddepcontrol.wait;" ::: "memory");
    for (int s = 0; s < kStages; ++s) {
      if (s > 0) {
        mbar_init(&bars->kfull[s], 1);
        mbar_init(&bars->vfull[s], 1);
      }
      mbar_init(&bars->pvfree[s], 1);
    }
    for (int b = 0; b < kSBuf; ++b) {
      mbar_init(&bars->sfull[b], 1);
      mbar_init(&bars->pfull[b], 8);  // one arrival per softmax warp
    }
    mbar_init(&bars->drain_s, 1);
    mbar_init(&bars->drain_pv, 1);
    mbar_init(&bars->qready, 8);
    mbar_init(&bars->tdone, 8);
    for (int qq = 0; qq < 4; ++qq) mbar_init(&bars->xchg[qq], 64);
    bars->abort = 0;
    bars->gen = p.gen;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 2) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(&bars->tmem_base)),
                 "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }

  fence_before();
  __syncthreads();
  fence_after();
  // The grid launched after this one (the branch/merge pass) may start its own
  // prologue now; it waits for this grid's completion before it reads partials.  With
  // the fused tail of a two-call step the next grid is the next step's append, which
  // must not overwrite partials that the tail still reads: no early release there.  The
  // next one-call step waits for this grid before it touches anything, so it may start.
  if (one_call || !p.fused) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const uint32_t tmem = bars->tmem_base;

  if (warp == 0 || warp == 3) {
    // ------------------------------------------------------------ TMA producers
    if (lane == 0) {
      const bool isK = warp == 0;
      const CUtensorMap* map = isK ? &tmK : &tmV;
      int issued = min(1, n_tiles);  // tile 0 went out in the prologue
      // the other stages fill once the first K tile has landed
      bool ok = n_tiles <= 1 || mbar_wait(&bars->kfull[0], 0u, bars, p.header, isK ? 1 : 2);
      for (int t = 1; t < n_tiles && ok; ++t) {
        const int s = t % kStages;
        if (t >= kStages) {
          // K stage: S of tile t-3 done (sfull[s], completion t/3 - 1); V stage: its P.V done
          uint64_t* freed = isK ? &bars->sfull[s] : &bars->pvfree[s];
          ok = mbar_wait(freed, (uint32_t)((t / kStages - 1) & 1), bars, p.header, isK ? 1 : 2);
          if (!ok) break;
        }
        uint64_t* full = isK ? &bars->kfull[s] : &bars->vfull[s];
        mbar_expect_tx(full, kTileBytes);
        const uint32_t dst = sbase + (isK ? kOffK : kOffV) + s * kTileBytes;
        tma_load_3d(dst, map, 0, kvh, tile_tok(t), full);
        tma_load_3d(dst + kHalfBytes, map, 64, kvh, tile_tok(t), full);
        issued = t + 1;
      }
      if (!ok) {
        // the loads already issued must land before the CTA leaves
        for (int t = max(0, issued - kStages); t < issued; ++t) {
          uint64_t* full = isK ? &bars->kfull[t % kStages] : &bars->vfull[t % kStages];
          drain_wait(full, (uint32_t)((t / kStages) & 1));
        }
      }
    }
    __syncwarp();
    if (!PREFILL && warp == 0 && !p.causal) prefetch_branch_tasks(p, q, kpool, vpool, lane);
  } else if (warp == 1 || warp == 2) {
    // ------------------------------------------------------------ MMA issuers
    // Two threads feed the tensor pipe so that one's waits and commits overlap the
    // other's MMAs: warp 1 issues S = Q K^T, warp 2 (after allocating TMEM) issues
    // O += P V.  A commit tracks only its own thread's MMAs, so each has its own
    // completion barriers (sfull / pvfree) and drain.
    if (lane == 0) {
      // Descriptors are built once; a K-step moves the start address, i.e. adds
      // (byte offset >> 4) to the low field (no carry: addresses stay below 256 KB).
      const uint64_t dQ = sdesc(sbase + kOffQ, 16, 1024);
      const uint64_t dK = sdesc(sbase + kOffK, 16, 1024);
      // V tile, N(=head-dim)-major: 16 tokens per step (2048 bytes), the second
      // 64-column half at +kHalfBytes (leading byte offset), 8-row groups 1024 apart.
      const uint64_t dV = sdesc(sbase + kOffV, kHalfBytes, 1024);
      bool ok = true;
      if (warp == 1) {
        ok = mbar_wait(&bars->qready, 0u, bars, p.header, 11);
        for (int t = 0; t < n_tiles && ok; ++t) {
          const uint32_t s = (uint32_t)(t % kStages);
          ok = mbar_wait(&bars->kfull[s], (uint32_t)((t / kStages) & 1), bars, p.header, 3);
          if (!ok) break;
          // S buffer s holds P of tile t-3 until that P.V completes
          if (t >= kStages)
            ok = mbar_wait(&bars->pvfree[s], (uint32_t)((t / kStages - 1) & 1), bars, p.header, 6);
          if (!ok) break;
          fence_after();
          const uint32_t d = tmem + 128u * s;
          const uint64_t kb = dK + (s * kTileBytes >> 4);
#pragma unroll
          for (int kk = 0; kk < kD / 16; ++kk) {
            const uint32_t off = (uint32_t)(kk >> 2) * kQHalfBytes + (uint32_t)(kk & 3) * 32;
            mma_ss(d, dQ + (off >> 4), kb + (off >> 4), kIdescS, kk > 0 ? 1u : 0u);
          }
          mma_commit(&bars->sfull[s]);
        }
        mma_commit(&bars->drain_s);
        drain_wait(&bars->drain_s, 0u);
      } else {
        for (int j = 0; j < n_tiles && ok; ++j) {
          const uint32_t s = (uint32_t)(j % kStages);
          ok = mbar_wait(&bars->vfull[s], (uint32_t)((j / kStages) & 1), bars, p.header, 4);
          if (!ok) break;
          ok = mbar_wait(&bars->pfull[s], (uint32_t)((j / kSBuf) & 1), bars, p.header, 5);
          if (!ok) break;
          fence_after();
          const uint32_t a = tmem + 128u * s;
          const uint64_t vb = dV + (s * kTileBytes >> 4);
          const uint32_t acc0 = j > 0 ? 1u : 0u;
#pragma unroll
          for (int kk = 0; kk < kBN / 16; ++kk)
            mma_ts(tmem + kColO, a + kk * 8, vb + ((uint32_t)kk * 2048 >> 4), kIdescPV,
                   kk > 0 ? 1u : acc0);
          mma_commit(&bars->pvfree[s]);
        }
        // O is final once every P.V has completed
        mma_commit(&bars->drain_pv);
        drain_wait(&bars->drain_pv, 0u);
      }
    }
  } else if (warp >= 4) {
    // ------------------------------------------------------------ softmax
    const int quarter = warp & 3;              // TMEM lanes 32*quarter .. +31 (query rows)
    const int half = (warp - 4) >> 2;          // rows 16*half .. +15 of the quarter
    const int lane_base = 32 * quarter;
    // Q rows (loaded in the prologue) into the 128-byte-swizzled K-major layout the
    // MMA reads: row r, 16-byte chunk cc of half h at h*16K + r*128 + ((cc ^ (r & 7)) << 4).
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int idx = lane + 32 * i;
      const int r = lane_base + (idx >> 3), cc = idx & 7;
      *reinterpret_cast<uint4*>(smem + kOffQ + half * kQHalfBytes + r * 128 + ((cc ^ (r & 7)) << 4)) = qv[i];
    }
    if (ROPE) {
      // Rotation in place: element d < 64 pairs with d + 64, i.e. chunk cc of half 0 with
      // chunk cc of half 1 of the same row, which the other warp of this lane quarter
      // stored.  The two warps meet (named barrier 2 + quarter) and split the quarter's
      // 32 rows x 8 chunk pairs; every table row is fetched once all four are addressed.
      asm volatile("bar.sync %0, 64;" ::"r"(2 + quarter) : "memory");
      const int t = half * 32 + lane;
      const float* cs[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int r = lane_base + ((t + 64 * i) >> 3);
        cs[i] = row0 + r < R
                    ? p.rope_cs + (size_t)plan_events(p)[it.first_event + (row0 + r) / p.group].pos * kD
                    : nullptr;
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        if (cs[i] == nullptr) continue;
        const int k = t + 64 * i;
        const int r = lane_base + (k >> 3), cc = k & 7;
        uint4* lo = reinterpret_cast<uint4*>(smem + kOffQ + r * 128 + ((cc ^ (r & 7)) << 4));
        uint4* hi = reinterpret_cast<uint4*>(smem + kOffQ + kQHalfBytes + r * 128 + ((cc ^ (r & 7)) << 4));
        const uint4 a = *lo, b = *hi;
        const float4 c0 = *reinterpret_cast<const float4*>(cs[i] + 8 * cc);
        const float4 c1 = *reinterpret_cast<const float4*>(cs[i] + 8 * cc + 4);
        const float4 s0 = *reinterpret_cast<const float4*>(cs[i] + 64 + 8 * cc);
        const float4 s1 = *reinterpret_cast<const float4*>(cs[i] + 64 + 8 * cc + 4);
        const float c[8] = {c0.x, c0.y, c0.z, c0.w, c1.x, c1.y, c1.z, c1.w};
        const float s[8] = {s0.x, s0.y, s0.z, s0.w, s1.x, s1.y, s1.z, s1.w};
        const uint32_t av[4] = {a.x, a.y, a.z, a.w}, bv[4] = {b.x, b.y, b.z, b.w};
        uint32_t ol[4], oh[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const float2 x = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&av[j]));
          const float2 y = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&bv[j]));
          const __nv_bfloat162 l2 = __floats2bfloat162_rn(rope_one(x.x, y.x, c[2 * j], s[2 * j], true),
                                                          rope_one(x.y, y.y, c[2 * j + 1], s[2 * j + 1], true));
          const __nv_bfloat162 h2 = __floats2bfloat162_rn(rope_one(y.x, x.x, c[2 * j], s[2 * j], false),
                                                          rope_one(y.y, x.y, c[2 * j + 1], s[2 * j + 1], false));
          ol[j] = *reinterpret_cast<const uint32_t*>(&l2);
          oh[j] = *reinterpret_cast<const uint32_t*>(&h2);
        }
        *lo = make_uint4(ol[0], ol[1], ol[2], ol[3]);
        *hi = make_uint4(oh[0], oh[1], oh[2], oh[3]);
      }
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    __syncwarp();
    if (lane == 0) mbar_arrive(&bars->qready);
    const float sl2 = p.scale_log2;
    bool ok = true;
    // Prefill: O leaves through shared memory, its rows staged in the K stages (idle once
    // every MMA has completed) at a padded stride, then normalised and written one 512-byte
    // row per warp instruction.  (One row per thread stored straight to global memory would
    // touch 32 lines per instruction; the decode layout stores straight, eight rows of 32
    // contiguous bytes per instruction.)
    float* ostage = reinterpret_cast<float*>(smem + kOffK);
    float* inv_row = ostage + 128 * kOStage;  // PREFILL: 1 / l of each row for the write-out
    if constexpr (PREFILL) {
      // columns 64*half .. +63 of every tile, one query row per thread
      const int row = lane_base + lane;
      const int grow = row0 + row;
      const bool warp_active = (row0 + lane_base) < R;  // same for both warps of the quarter
      const uint32_t tl = tmem + ((uint32_t)lane_base << 16);
      const uint32_t col0 = 64u * (uint32_t)half;
      float* xmax = reinterpret_cast<float*>(smem + kOffX);  // [tile parity][half][row]
      uint64_t* xbar = &bars->xchg[quarter];
      float m_run = -__builtin_huge_valf(), l_run = 0.f;
      uint32_t r[32];
      // this row's token and the first token of its branch (-1 in the prefix)
      int pf_p = 0, pf_bs = -1;
      if (grow < R) {
        pf_p = it.first_event + grow / p.group;
        pf_bs = pf_p >= p.pf_S ? pf_branch_start(p, pf_p) : -1;
      }
      for (int j = 0; j < n_tiles; ++j) {
        const uint32_t cS = 128u * (uint32_t)(j % kSBuf);
        ok = mbar_wait(&bars->sfull[j % kSBuf], (uint32_t)((j / kSBuf) & 1), bars, p.header, 8);
        ok = __all_sync(0xffffffffu, ok);  // tcgen05.ld/st below are warp-collective
        if (!ok) break;
        fence_after();
        if (warp_active) {
          uint32_t sr[2][32];
          tmem_ld32(tl + cS + col0, sr[0]);
          tmem_ld32(tl + cS + col0 + 32, sr[1]);
          tmem_wait_ld_dep(sr[0]);
          tmem_wait_ld_dep(sr[1]);
          // the tile's range end, then this row's rule: a prefix token sees keys up to
          // itself, a branch token the prefix and its own branch up to itself
          const int tb = tile_tok(j);
          const int t0 = tb + (int)col0;
          uint64_t keep = range_bits(0, min(kBN, (j < pf_a_tiles ? pf_a_end : pf_last + 1) - tb) - (int)col0);
          if (grow < R)
            keep &= pf_bs < 0 ? range_bits(0, pf_p - t0 + 1)
                              : (range_bits(0, p.pf_S - t0) | range_bits(pf_bs - t0, pf_p - t0 + 1));
          const bool masked = __any_sync(0xffffffffu, keep != ~0ull);
          const float pmax = masked ? half_row_max<true>(sr, HalfBits{keep}) : half_row_max<false>(sr, HalfBits{keep});
          // meet the other half: this also orders both warps' S reads before either
          // writes P over columns the other one read
          xmax[(j & 1) * 256 + half * 128 + row] = pmax;
          mbar_arrive(xbar);
          ok = mbar_wait(xbar, (uint32_t)(j & 1), bars, p.header, 12);
          ok = __all_sync(0xffffffffu, ok);
          if (!ok) break;
          const float mx = fmaxf(pmax, xmax[(j & 1) * 256 + (1 - half) * 128 + row]) * sl2;
          const float m_new = fmaxf(m_run, mx);
          const bool need = m_new > m_run + kLazyRescale;
          if (__any_sync(0xffffffffu, need && j > 0)) {
            // O must hold P.V of tile j-1 before it is rescaled (each half rescales its
            // own 64 head-dim columns; both halves take the same decision per row)
            ok = mbar_wait(&bars->pvfree[(j - 1) % kStages], (uint32_t)(((j - 1) / kStages) & 1), bars,
                           p.header, 9);
            ok = __all_sync(0xffffffffu, ok);
            if (!ok) break;
            fence_after();
            const float alpha = need ? ex2(m_run - m_new) : 1.f;
#pragma unroll
            for (int c = 0; c < 2; ++c) {
              tmem_ld32(tl + kColO + col0 + 32 * c, r);
              tmem_wait_ld_dep(r);
#pragma unroll
              for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * alpha);
              tmem_st32(tl + kColO + col0 + 32 * c, r);
            }
            tmem_wait_st();
            if (need) l_run *= alpha;
          }
          if (need) m_run = m_new;
          l_run += masked ? half_row_exp<true>(sr, HalfBits{keep}, sl2, m_run, tl + cS + col0 / 2)
                          : half_row_exp<false>(sr, HalfBits{keep}, sl2, m_run, tl + cS + col0 / 2);
          tmem_wait_st();
        }
        fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars->pfull[j % kSBuf]);
      }
      // the P.V issuer commits `drain_pv` after its last MMA: O is final once it lands
      if (ok) ok = mbar_wait(&bars->drain_pv, 0u, bars, p.header, 10);
      ok = __all_sync(0xffffffffu, ok);
      if (ok && warp_active) {
        fence_after();
#pragma unroll
        for (int c = 0; c < 2; ++c) {
          tmem_ld32(tl + kColO + col0 + 32 * c, r);
          tmem_wait_ld_dep(r);
          float4* dst = reinterpret_cast<float4*>(ostage + row * kOStage + col0 + 32 * c);
#pragma unroll
          for (int i = 0; i < 8; ++i)
            dst[i] = make_float4(__uint_as_float(r[4 * i]), __uint_as_float(r[4 * i + 1]),
                                 __uint_as_float(r[4 * i + 2]), __uint_as_float(r[4 * i + 3]));
        }
        // row sum = both halves' partial sums (slot n_tiles & 1 was last read two tiles ago)
        xmax[(n_tiles & 1) * 256 + half * 128 + row] = l_run;
        mbar_arrive(xbar);
        ok = mbar_wait(xbar, (uint32_t)(n_tiles & 1), bars, p.header, 13);
        if (ok && half == 0 && grow < R) {
          // normalised output: 1 / l for the write-out below, the LSE now
          const float l_tot = l_run + xmax[(n_tiles & 1) * 256 + 128 + row];
          inv_row[row] = 1.0f / l_tot;
          const int64_t orow = (int64_t)pf_p * p.h_q + kvh * p.group + grow % p.group;
          if (p.pf_lse != nullptr) p.pf_lse[orow] = (m_run + log2f(l_tot)) * 0.69314718055994531f;
        }
      }
    } else {
      // this warp's 16 rows (TMEM lanes), this thread's two of them and its first column of
      // every 8-column chunk
      const int wrow = lane_base + 16 * half;
      const int ra = wrow + (lane >> 2), rb = ra + 8;
      const int ga = row0 + ra, gb = row0 + rb;
      const int cq = 2 * (lane & 3);
      const bool warp_active = (row0 + wrow) < R;
      const uint32_t tl = tmem + ((uint32_t)wrow << 16);
      float m_a = -__builtin_huge_valf(), m_b = -__builtin_huge_valf(), l_a = 0.f, l_b = 0.f;
      // self G-token mask: the video's planning tokens G^1..G^K (prefix-relative [g_lo, g_hi))
      // and each row's own one
      int g_lo = 0, g_hi = 0, g_oa = -1, g_ob = -1;
      if (GSELF) {
        const PadVideoDesc vdg = plan_videos(p)[plan_events(p)[it.first_event].video];
        if (vdg.n_planning > 0) {
          g_lo = vdg.prefix_len - 1 - vdg.n_planning;
          g_hi = vdg.prefix_len - 1;
          if (ga < R) g_oa = g_lo + plan_events(p)[it.first_event + ga / p.group].gidx;
          if (gb < R) g_ob = g_lo + plan_events(p)[it.first_event + gb / p.group].gidx;
        }
      }
      uint32_t sr[2][32];
      for (int j = 0; j < n_tiles; ++j) {
        const uint32_t cS = 128u * (uint32_t)(j % kSBuf);
        ok = mbar_wait(&bars->sfull[j % kSBuf], (uint32_t)((j / kSBuf) & 1), bars, p.header, 8);
        ok = __all_sync(0xffffffffu, ok);  // tcgen05.ld/st below are warp-collective
        if (!ok) break;
        fence_after();
        if (warp_active) {
          const int valid = min(kBN, ntok - j * kBN);  // valid columns of the tile
          tmem_ld16x256_x8(tl + cS, sr[0]);
          tmem_ld16x256_x8(tl + cS + 64, sr[1]);
          tmem_wait_ld_dep(sr[0]);
          tmem_wait_ld_dep(sr[1]);
          // columns to mask: past the split's end, or (GSELF) hidden planning tokens of the
          // row's event; the path is chosen per warp (tcgen05.st below is warp-collective)
          float mxa, mxb;
          bool masked;
          ColsBits ka{~0ull, ~0ull}, kb{~0ull, ~0ull};
          if (GSELF) {
            const int t0 = it.tok_begin + j * kBN;
            if (valid < kBN || (t0 < g_hi && t0 + kBN > g_lo)) {
              const GMask gma{g_lo, g_hi, g_oa}, gmb{g_lo, g_hi, g_ob};
              ka = ColsBits{keep_bits(valid, gma, t0), keep_bits(valid - 64, gma, t0 + 64)};
              kb = ColsBits{keep_bits(valid, gmb, t0), keep_bits(valid - 64, gmb, t0 + 64)};
            }
            masked = __any_sync(0xffffffffu, (ka.lo & ka.hi & kb.lo & kb.hi) != ~0ull);
            if (masked) rows_max<true>(sr, cq, ka, kb, mxa, mxb);
            else rows_max<false>(sr, cq, ka, kb, mxa, mxb);
          } else {
            masked = valid < kBN;
            if (masked) rows_max<true>(sr, cq, ColsValid{valid}, ColsValid{valid}, mxa, mxb);
            else rows_max<false>(sr, cq, ColsValid{valid}, ColsValid{valid}, mxa, mxb);
          }
          const float na = fmaxf(m_a, mxa * sl2), nb = fmaxf(m_b, mxb * sl2);
          const bool need_a = na > m_a + kLazyRescale, need_b = nb > m_b + kLazyRescale;
          if (__any_sync(0xffffffffu, (need_a || need_b) && j > 0)) {
            // O must hold P.V of tile j-1 before its rows are rescaled
            ok = mbar_wait(&bars->pvfree[(j - 1) % kStages], (uint32_t)(((j - 1) / kStages) & 1), bars,
                           p.header, 9);
            ok = __all_sync(0xffffffffu, ok);
            if (!ok) break;
            fence_after();
            const float al_a = need_a ? ex2(m_a - na) : 1.f, al_b = need_b ? ex2(m_b - nb) : 1.f;
#pragma unroll
            for (int x = 0; x < 2; ++x) {
              uint32_t o[32];
              tmem_ld16x256_x8(tl + kColO + 64 * x, o);
              tmem_wait_ld_dep(o);
#pragma unroll
              for (int i = 0; i < 32; ++i)
                o[i] = __float_as_uint(__uint_as_float(o[i]) * ((i & 2) ? al_b : al_a));
              tmem_st16x256_x8(tl + kColO + 64 * x, o);
            }
            tmem_wait_st();
            l_a *= al_a;
            l_b *= al_b;
          }
          if (need_a) m_a = na;
          if (need_b) m_b = nb;
          // P of the tile over the first 64 columns of its S buffer, in this warp's own rows
          if (GSELF) {
            if (masked) rows_exp<true>(sr, cq, ka, kb, sl2, m_a, m_b, tl + cS, l_a, l_b);
            else rows_exp<false>(sr, cq, ka, kb, sl2, m_a, m_b, tl + cS, l_a, l_b);
          } else {
            if (masked) rows_exp<true>(sr, cq, ColsValid{valid}, ColsValid{valid}, sl2, m_a, m_b, tl + cS, l_a, l_b);
            else rows_exp<false>(sr, cq, ColsValid{valid}, ColsValid{valid}, sl2, m_a, m_b, tl + cS, l_a, l_b);
          }
          tmem_wait_st();
        }
        fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars->pfull[j % kSBuf]);
      }
      // the P.V issuer commits `drain_pv` after its last MMA: O is final once it lands
      if (ok) ok = mbar_wait(&bars->drain_pv, 0u, bars, p.header, 10);
      ok = __all_sync(0xffffffffu, ok);
      if (ok && warp_active) {
        fence_after();
        // O rows straight from the 16-lane layout: a quad writes 32 contiguous bytes of a
        // row, a warp instruction eight such segments
        float* po_a = p.part_o + ((int64_t)it.part_row0 + ga) * kD;
        float* po_b = po_a + 8 * kD;
#pragma unroll
        for (int x = 0; x < 2; ++x) {
          uint32_t o[32];
          tmem_ld16x256_x8(tl + kColO + 64 * x, o);
          tmem_wait_ld_dep(o);
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const int c = 64 * x + 8 * k + cq;
            if (ga < R)
              *reinterpret_cast<float2*>(po_a + c) = make_float2(__uint_as_float(o[4 * k]), __uint_as_float(o[4 * k + 1]));
            if (gb < R)
              *reinterpret_cast<float2*>(po_b + c) =
                  make_float2(__uint_as_float(o[4 * k + 2]), __uint_as_float(o[4 * k + 3]));
          }
        }
        const float la = quad_sum(l_a), lb = quad_sum(l_b);
        if ((lane & 3) == 0) {
          if (ga < R) p.part_ml[(int64_t)it.part_row0 + ga] = make_float2(m_a, la);
          if (gb < R) p.part_ml[(int64_t)it.part_row0 + gb] = make_float2(m_b, lb);
        }
      }
    }
    // TMEM is freed by warp 2 only after every softmax warp has arrived here
    fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive(&bars->tdone);
    // every softmax warp reaches this barrier exactly once (the loop above only breaks);
    // it orders the staged rows (prefill) and the partial rows before the fused tail
    if (PREFILL || p.fused) asm volatile("bar.sync 1, 256;" ::: "memory");
    const int nrows = PREFILL ? min(128, R - row0) : 0;  // prefill: normalised rows out
    for (int rr = warp - 4; rr < nrows; rr += 8) {
      float4 v = *reinterpret_cast<const float4*>(ostage + rr * kOStage + 4 * lane);
      const float inv = inv_row[rr];
      v.x *= inv;
      v.y *= inv;
      v.z *= inv;
      v.w *= inv;
      const int gr = row0 + rr;
      const size_t oi = ((size_t)(it.first_event + gr / p.group) * p.h_q + kvh * p.group + gr % p.group) * kD + 4 * lane;
      if (p.out_bf16)
        *reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(p.pf_out) + oi) =
            make_uint2(bm::pack_bf16(v.x, v.y), bm::pack_bf16(v.z, v.w));
      else
        *reinterpret_cast<float4*>(static_cast<float*>(p.pf_out) + oi) = v;
    }
    if (!PREFILL && p.fused) {
      // ---------------------------------------------------------- fused a4 + a5
      // Publish this split's rows (every softmax thread's partial stores are ordered
      // before the counter by the barrier and the fence), then run this CTA's (event,
      // kv-head) task with all of shared memory below the barriers (the Q, K and V
      // stages are idle once the last MMA has completed).
      const bm::SyncNamed sy{1};
      if (sy.all(ok)) {
        if (threadIdx.x == 128) {
          // the append kernel ahead zeroes the counters: wait for it (long complete by now)
          asm volatile("griddepcontrol.wait;" ::: "memory");
          __threadfence();
          const PadVideoDesc vd = plan_videos(p)[plan_events(p)[it.first_event].video];
          atomicAdd(p.counters + vd.cnt_base + (size_t)kvh * ((R + 127) >> 7) + group, 1u);
        }
        const int task = plan_tasks(p)[blockIdx.x];
        if (task >= 0) {
          const int te = task / p.h_kv, th = task - (task / p.h_kv) * p.h_kv;
          bm::run_task<kD, ROPE, 2>(p, q, kpool, vpool, out, lse, te, th, (int)threadIdx.x - 128, smem, p.tail_chunk, sy,
                           false, [&]() {
                             const PadEventDesc ev = plan_events(p)[te];
                             const PadVideoDesc vd = plan_videos(p)[ev.video];
                             return tail_partials_ready(p, vd, th, ev.local * p.group, threadIdx.x == 128);
                           });
        }
      }
    }
  }

  __syncwarp();
  fence_before();
  // This grid may run alongside the append kernel before it (it reads nothing that
  // kernel writes); waiting for it here makes the completion of this grid imply the
  // completion of the append, which the branch/merge pass after it relies on.
  if (threadIdx.x == 0) asm volatile("griddepcontrol.wait;" ::: "memory");
  __syncthreads();
  if (warp == 2) {
    // The block barrier above is not relied on to order the softmax warps' last TMEM
    // reads before the deallocation (it was measured to let the role warps through
    // before them); their own arrivals are.
    drain_wait(&bars->tdone, 0u);
    fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols)
                 : "memory");
  }
}

PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult qres;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &qres) == cudaSuccess &&
        qres == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  }
  return fn;
}

// Token-major [T, h_kv, 128] bf16 prefix as a 3-D tensor (d, head, token); one box is
// 64 head-dim columns x 1 head x 128 tokens with the 128-byte swizzle.
bool make_map(CUtensorMap* map, const void* base, int h_kv, int64_t tokens) {
  auto enc = get_encode();
  if (!enc) return false;
  cuuint64_t dims[3] = {(cuuint64_t)kD, (cuuint64_t)h_kv, (cuuint64_t)tokens};
  cuuint64_t strides[2] = {(cuuint64_t)kD * 2, (cuuint64_t)h_kv * kD * 2};
  cuuint32_t box[3] = {64, 1, (cuuint32_t)kBN};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides,
                   box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// The tensor maps of the last few (K, V) prefix buffers, so a step does not re-encode
// them (an encode costs microseconds of host time; the maps depend only on the base
// address, the head count and the token extent).
struct MapCacheEntry {
  const void* k;
  const void* v;
  int h_kv;
  int64_t tokens;
  int dev;
  CUtensorMap mk, mv;
};
std::mutex g_map_mu;
MapCacheEntry g_maps[8];
int g_maps_n = 0, g_maps_next = 0;

}  // namespace

bool prefix_tensor_maps(const void* kp, const void* vp, int h_kv, int64_t tokens, int dev, CUtensorMap* mk,
                        CUtensorMap* mv) {
  std::lock_guard<std::mutex> lk(g_map_mu);
  for (int i = 0; i < g_maps_n; ++i) {
    const MapCacheEntry& e = g_maps[i];
    if (e.k == kp && e.v == vp && e.h_kv == h_kv && e.tokens == tokens && e.dev == dev) {
      std::memcpy(mk, &e.mk, sizeof(CUtensorMap));
      std::memcpy(mv, &e.mv, sizeof(CUtensorMap));
      return true;
    }
  }
  MapCacheEntry ne;
  ne.k = kp;
  ne.v = vp;
  ne.h_kv = h_kv;
  ne.tokens = tokens;
  ne.dev = dev;
  if (!make_map(&ne.mk, kp, h_kv, tokens) || !make_map(&ne.mv, vp, h_kv, tokens)) return false;
  g_maps[g_maps_next] = ne;
  g_maps_next = (g_maps_next + 1) % 8;
  if (g_maps_n < 8) ++g_maps_n;
  std::memcpy(mk, &ne.mk, sizeof(CUtensorMap));
  std::memcpy(mv, &ne.mv, sizeof(CUtensorMap));
  return true;
}

int prefix_tc_tail_chunk(int branch_rows, int group, int max_splits) {
  int sch = std::min(bm::kMaxChunk, std::max(1, max_splits));
  while (sch > 1 && bm::smem_bytes<kD>(branch_rows, group, sch) > kOffBar) --sch;
  return sch;
}

cudaError_t launch_prefix_tc(const KParams& p, int max_rows, const void* q, const void* kp,
                             const void* vp, int64_t total_prefix_tokens, const void* k_pool,
                             const void* v_pool, void* out, float* lse, bool pdl, cudaStream_t s) {
  if (p.n_items == 0) return cudaSuccess;
  if (p.head_dim != kD || total_prefix_tokens <= 0 || total_prefix_tokens > (int64_t)INT32_MAX)
    return cudaErrorInvalidValue;
  int dev = 0;
  cudaGetDevice(&dev);
  CUtensorMap mk, mv;
  if (!prefix_tensor_maps(kp, vp, p.h_kv, total_prefix_tokens, dev, &mk, &mv)) return cudaErrorInvalidValue;
  static bool configured[64] = {};
  if (dev >= 0 && dev < 64 && !configured[dev]) {
    for (auto fn : {prefix_tc_kernel<false, false, false>, prefix_tc_kernel<true, false, false>,
                    prefix_tc_kernel<false, true, false>, prefix_tc_kernel<true, true, false>}) {
      cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
      if (e != cudaSuccess) return e;
    }
    configured[dev] = true;
  }
  const int n_groups = (max_rows + 127) / 128;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.cta_map ? p.n_ctas : p.n_items * n_groups);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = kSmemBytes;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (p.fused && bm::smem_bytes<kD>(p.branch_rows, p.group, p.tail_chunk) > kOffBar) return cudaErrorInvalidValue;
  auto fn = p.rope_cs != nullptr
                ? (p.g_self ? prefix_tc_kernel<true, true, false> : prefix_tc_kernel<true, false, false>)
                : (p.g_self ? prefix_tc_kernel<false, true, false> : prefix_tc_kernel<false, false, false>);
  return cudaLaunchKernelEx(&cfg, fn, p, static_cast<const __nv_bfloat16*>(q), n_groups, mk, mv,
                            static_cast<const __nv_bfloat16*>(k_pool), static_cast<const __nv_bfloat16*>(v_pool),
                            out, lse);
}

// Device status word of the whole-sequence prefill (no plan or workspace is involved).
__device__ PadDevHeader g_prefill_header;

cudaError_t prefill_header(PadDevHeader** out) {
  static PadDevHeader* ptr[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (!ptr[dev]) {
    void* a = nullptr;
    e = cudaGetSymbolAddress(&a, g_prefill_header);
    if (e != cudaSuccess) return e;
    ptr[dev] = static_cast<PadDevHeader*>(a);
  }
  *out = ptr[dev];
  return cudaSuccess;
}

cudaError_t launch_prefill_tc(int32_t n_tokens, int32_t prefix_len, int32_t n_branches, const int32_t* branch_len,
                              int32_t h_q, int32_t h_kv, float scale, int32_t out_bf16, uint64_t gen, const void* q,
                              const void* k, const void* v, void* out, float* lse, cudaStream_t s) {
  const int G = h_q / h_kv;
  if (G < 1 || G > 128 || n_tokens <= 0) return cudaErrorInvalidValue;
  if ((size_t)(n_branches + 1) * sizeof(int32_t) > sizeof(KParams::img)) return cudaErrorInvalidValue;
  int dev = 0;
  cudaGetDevice(&dev);
  CUtensorMap mk, mv;
  if (!prefix_tensor_maps(k, v, h_kv, n_tokens, dev, &mk, &mv)) return cudaErrorInvalidValue;
  static bool configured[64] = {};
  if (dev >= 0 && dev < 64 && !configured[dev]) {
    cudaError_t e = cudaFuncSetAttribute(prefix_tc_kernel<false, false, true>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
    if (e != cudaSuccess) return e;
    configured[dev] = true;
  }
  KParams p;
  std::memset(&p, 0, offsetof(KParams, img));
  p.h_q = h_q;
  p.h_kv = h_kv;
  p.group = G;
  p.head_dim = kD;
  p.out_bf16 = out_bf16;
  p.scale_log2 = (float)((double)scale * 1.4426950408889634);
  p.gen = gen;
  cudaError_t e = prefill_header(&p.header);
  if (e != cudaSuccess) return e;
  p.pf_N = n_tokens;
  p.pf_S = prefix_len;
  p.pf_nb = n_branches;
  p.pf_tpc = 128 / G;
  p.pf_out = out;
  p.pf_lse = lse;
  int32_t* bs = reinterpret_cast<int32_t*>(p.img);
  bs[0] = prefix_len;
  for (int b = 0; b < n_branches; ++b) bs[b + 1] = bs[b] + branch_len[b];
  const int n_qt = (n_tokens + p.pf_tpc - 1) / p.pf_tpc;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(n_qt * h_kv);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = kSmemBytes;
  cfg.stream = s;
  cfg.numAttrs = 0;
  return cudaLaunchKernelEx(&cfg, prefix_tc_kernel<false, false, true>, p, static_cast<const __nv_bfloat16*>(q), 1,
                            mk, mv, static_cast<const __nv_bfloat16*>(nullptr),
                            static_cast<const __nv_bfloat16*>(nullptr), static_cast<void*>(nullptr),
                            static_cast<float*>(nullptr));
}

}  // namespace pad
