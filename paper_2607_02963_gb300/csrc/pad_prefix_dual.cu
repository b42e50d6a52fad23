// a3 on the 5th-generation tensor cores, with two softmax groups per CTA: split-KV
// flash-decode over the shared prefix (the part of the event-factorized mask of Sec. 3.4
// that every branch of a video sees: the multimodal prefix P and all planning tokens
// G^1..G^K, S).
//
// One CTA per (work item = video, kv-head, prefix split; group of <= 256 query rows).
// The CTA has two slots, each with its own S buffer and O accumulator in TMEM and its own
// softmax warpgroup, so that one slot's softmax runs while the tensor pipe works for the
// other (the two alternate):
//   rows  > 128: slot g holds query rows 128g .. 128g+127 of the CTA; every K/V tile
//                brought from HBM serves both (S_g = Q_g K^T, O_g += P_g V), so a tile
//                enters one SM once for up to 256 rows (for 224 rows: 7 events x 7 heads
//                of GQA 28/4 x 32 events);
//   rows <= 128: both slots hold the same rows and take alternate tiles (slot = tile
//                parity); the two partial softmax states are merged at the end.
//
//   warp 0      TMA producer (one thread): K tiles into a 3-stage ring, V tiles into 2
//               stages (3 with one row group, whose second Q buffer is then free);
//               128-token tiles as two 64-column boxes with the 128-byte swizzle.  After
//               its last tile it prefetches the branch data of one (event, kv-head) task
//               into L2 for the branch pass that follows.
//   warp 1      S issuer (one thread): S_g(k) = Q_g K^T of the slot's k-th tile into S_g,
//               once the P.V of the slot's previous tile (whose P lives in S_g) completed
//   warp 2      TMEM allocation (512 columns: S_0, S_1, O_0, O_1) and deallocation; its
//               lane 0 issues O_g += P_g(k) V with P read back from TMEM
//   warps 4-7   softmax of slot 0, warps 8-11 of slot 1: one query row per thread, all 128
//               columns of a tile; online maximum and sum in base 2; P written as packed
//               bf16 over the S columns already read; O rescaled only when a row maximum
//               grows by more than 2^8.  Each group then writes its slot's partial state
//               (m, l, O) through shared memory.
//
// Output: the partial softmax state (m, l, O) of every row for this split, in the layout
// the branch/merge kernel merges with the other splits and the branch (rows of an item
// are contiguous from its part_row0).
//
// Every mbarrier wait is bounded (about one second of %globaltimer); a wait that runs out
// records PAD_ERR_DEVICE_TIMEOUT in the status word, raises a CTA-wide abort flag, lets the
// producer and the MMA issuer drain what they already started, frees TMEM and returns.
// Barrier phases: each barrier is per slot or per stage, so the completion a thread waits
// for by parity cannot be overtaken by the next one before the thread itself moves on.
#include <cuda.h>
#include <cuda_bf16.h>
#include <algorithm>
#include <cstddef>
#include <cstdint>

#include "pad_internal.h"
#include "pad_tc_common.cuh"

namespace pad {

namespace {

using namespace tc;

constexpr int kD = 128;
constexpr int kBN = 128;                           // prefix tokens per K/V tile
constexpr int kKS = 3;                             // K stages
constexpr int kThreads = 384;
constexpr uint32_t kHalfBytes = kBN * 128;         // 128 tokens x 64 bf16 = 16 KB
constexpr uint32_t kTileBytes = 2 * kHalfBytes;    // one K (or V) tile: 32 KB
constexpr uint32_t kQHalfBytes = 128 * 128;        // 128 rows x 64 bf16 = 16 KB
constexpr uint32_t kQTileBytes = 2 * kQHalfBytes;  // Q of one slot: 32 KB
// Shared memory: [Q_0 | Q_1 or V stage 2 | K stages 0-2 | V stages 0-1 | barriers | row states]
constexpr uint32_t kOffQ0 = 0;
constexpr uint32_t kOffQ1 = kQTileBytes;
constexpr uint32_t kOffK = 2 * kQTileBytes;
constexpr uint32_t kOffV = kOffK + kKS * kTileBytes;
constexpr uint32_t kOffBar = kOffV + 2 * kTileBytes;
constexpr uint32_t kOffX = kOffBar + 512;          // (m, l) of both slots' rows: float2 [2][128]
constexpr uint32_t kSmemBytes = kOffX + 2 * 128 * 8;
static_assert(kSmemBytes <= 232448, "fits the 227 KB opt-in shared memory");
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColO = 256;                    // O_g at kColO + 128 g; S_g at 128 g
constexpr float kLazyRescale = 8.0f;               // log2 units
// One exponential pair in every kPolyEvery goes to exp2_poly2 on the FMA pipe instead of the
// MUFU unit (0: none).  The softmax of one slot has 128 x 128 exponentials per tile, which
// at 16 per clock and SM take about as long as the tensor pipe spends on both slots' MMAs.
#ifdef PAD_DUAL_POLY_EVERY
constexpr int kPolyEvery = PAD_DUAL_POLY_EVERY;
#else
constexpr int kPolyEvery = 0;
#endif
constexpr uint32_t kIdescS = make_idesc(128, kBN, false);   // S = Q K^T: B = K tile, K-major
constexpr uint32_t kIdescPV = make_idesc(128, kD, true);    // O += P V: B = V tile, N(=d)-major

struct DualBars {
  uint64_t kfull[kKS];
  uint64_t kfree[kKS];        // the S MMAs of the tile in this stage have completed
  uint64_t vfull[3];
  uint64_t vfree[3];          // the P.V MMAs of the tile in this stage have completed
  uint64_t sfull[2];          // S of the slot's current tile has completed
  uint64_t plo[2];            // P of the first half of the slot's current tile is written
                              // (4 warp arrivals)
  uint64_t phi[2];            // P of its second half is written (4 warp arrivals)
  uint64_t pvlo[2];           // P.V of the first half of the slot's current tile has completed
  uint64_t pvdone[2];         // P.V of the slot's current tile has completed
  uint64_t drain_s;           // every S MMA has completed (end of the S issuer)
  uint64_t drain_pv;          // every P.V MMA has completed (end of the P.V issuer)
  uint64_t qready;            // Q staged in shared memory (8 warp arrivals)
  uint64_t tdone;             // the softmax warps are done with TMEM (8 warp arrivals)
  uint64_t gen;               // the plan's generation, for the status word
  uint32_t tmem_base;
  int32_t abort;
};
static_assert(sizeof(DualBars) <= 512, "barrier block fits its slot");

// Bounded wait (as mbar_wait_b), with the slow path inlined.
__device__ __forceinline__ bool dwait(uint64_t* bar, uint32_t parity, DualBars* bars, PadDevHeader* hdr, int where) {
  if (mbar_try_wait(bar, parity)) return true;
  const unsigned long long t0 = globaltimer();
  for (uint32_t i = 1;; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 63u) == 0) {
      if (*reinterpret_cast<volatile int32_t*>(&bars->abort)) return false;
      if (globaltimer() - t0 > kWaitNs) {
        pad_set_error(hdr, bars->gen, PAD_ERR_DEVICE_TIMEOUT, (int)blockIdx.x, where, (int)threadIdx.x);
        *reinterpret_cast<volatile int32_t*>(&bars->abort) = 1;
        return false;
      }
    }
  }
}


// Shared-memory offset of V stage s (stage 2 exists with one row group only).
__device__ __forceinline__ uint32_t v_off(int s) { return s < 2 ? kOffV + (uint32_t)s * kTileBytes : kOffQ1; }

// The softmax works on half rows: 64 raw scores of one thread (two 32-column TMEM loads).

// Hidden columns of a half row (bit c of keep clear) to -inf: they then get P = 0 and no
// say in the maximum.
__device__ __forceinline__ void mask_half(uint32_t (&h)[2][32], uint64_t keep) {
#pragma unroll
  for (int c = 0; c < 2; ++c)
#pragma unroll
    for (int i = 0; i < 32; ++i)
      if (!((keep >> (32 * c + i)) & 1ull)) h[c][i] = 0xff800000u;  // -inf
}

// P = 2^(s * sl2 - m) for a half row, packed two bf16 per word into pk[32] (tokens 2j and
// 2j + 1 in word j).  Returns the fp32 sum of the P values and, in *mx, the maximum of the
// raw scores, so that one pass both uses the running maximum and checks that it still
// bounds this half.
__device__ __forceinline__ float half_exp(const uint32_t (&h)[2][32], float sl2, float m, uint32_t (&pk)[32],
                                          float* mx) {
  const uint64_t sc2 = f2pack(sl2, sl2), nm2 = f2pack(-m, -m);
  uint64_t lacc[4] = {0ull, 0ull, 0ull, 0ull};
  float mt[4] = {-__builtin_huge_valf(), -__builtin_huge_valf(), -__builtin_huge_valf(), -__builtin_huge_valf()};
#pragma unroll
  for (int c = 0; c < 2; ++c)
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const float s0 = __uint_as_float(h[c][2 * i]), s1 = __uint_as_float(h[c][2 * i + 1]);
      const uint64_t x = ffma2(f2pack(s0, s1), sc2, nm2);
      float p0, p1;
      if (kPolyEvery == 0 || (i % kPolyEvery) != kPolyEvery - 1) {
        p0 = ex2(f2lo(x));
        p1 = ex2(f2hi(x));
      } else {
        const uint64_t e = exp2_poly2(x);
        p0 = f2lo(e);
        p1 = f2hi(e);
      }
      mt[i & 3] = max3f(mt[i & 3], s0, s1);
      lacc[i & 3] = fadd2(lacc[i & 3], f2pack(p0, p1));
      pk[16 * c + i] = pack_bf16(p0, p1);
    }
  *mx = fmaxf(fmaxf(mt[0], mt[1]), fmaxf(mt[2], mt[3]));
  const uint64_t ls = fadd2(fadd2(lacc[0], lacc[1]), fadd2(lacc[2], lacc[3]));
  return f2lo(ls) + f2hi(ls);
}

// Bits c of [0, 64) with c < n (clamped).
__device__ __forceinline__ uint64_t low_bits(int n) {
  return n >= 64 ? ~0ull : (n <= 0 ? 0ull : ((1ull << n) - 1ull));
}

// Staging of a slot's O rows for the write-out: row r (of 128) at r * 512 bytes, its 16-byte
// chunk c (of 32) at chunk position c ^ (r & 31), so that a warp writing chunk c of 32
// consecutive rows, and a warp reading all chunks of one row, touch distinct banks.
__device__ __forceinline__ uint32_t stage_off(int r, int c) { return (uint32_t)r * 512u + (uint32_t)((c ^ (r & 31)) << 4); }

// ---------------------------------------------------------------- kernel
template <bool ROPE, bool GSELF>
__global__ void __launch_bounds__(kThreads, 1)
    prefix_dual_kernel(const __grid_constant__ KParams p, const __nv_bfloat16* __restrict__ q, const int n_groups,
                       const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                       const __nv_bfloat16* __restrict__ kpool, const __nv_bfloat16* __restrict__ vpool) {
  extern __shared__ __align__(1024) uint8_t smem[];
  const uint32_t sbase = smem_u32(smem);
  if (sbase & 1023u) {  // the 128-byte swizzle atoms need 1024-byte alignment (never expected)
    if (threadIdx.x == 0) pad_set_error(p.header, p.gen, PAD_ERR_UNSUPPORTED, (int)blockIdx.x, (int)sbase, 1);
    return;
  }
  DualBars* bars = reinterpret_cast<DualBars*>(smem + kOffBar);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // One-call step (k_new set): this is the step's first kernel, launched so that it may
  // start while the grid before it finishes; every thread that touches global memory
  // waits for that grid first (the Q loads, the first TMA issue).
  const bool one_call = p.k_new != nullptr;

  // the CTA's work item and 256-row group: from the plan's CTA list, or the dense grid
  int item, grp;
  if (p.cta_map) {
    const int v = plan_tasks(p)[blockIdx.x];
    item = v >> 6;
    grp = v & 63;
  } else {
    item = blockIdx.x / n_groups;
    grp = blockIdx.x - item * n_groups;
  }
  const PadWorkItem it = plan_items(p)[item];
  const int R = it.n_events * p.group;
  const int row0 = grp * 256;
  if (row0 >= R) return;  // uniform over the CTA, before any barrier or allocation
  const int rows = min(256, R - row0);
  const bool dual = rows > 128;            // two row groups; else one row group, tiles by parity
  const int VS = dual ? 2 : 3;             // V stages
  const int ntok = it.tok_end - it.tok_begin;
  const int n_tiles = (ntok + kBN - 1) / kBN;
  const int kvh = it.kvh;
  const int tok0 = (int)it.tok0;
  const int n_slot0 = dual ? n_tiles : (n_tiles + 1) / 2;
  const int n_slot1 = dual ? n_tiles : n_tiles / 2;
  // Slot-tiles in issue order: i -> slot i & 1, the slot's (i >> 1)-th tile, which is tile
  // i >> 1 with two row groups and tile i with one.
  const int n_seq = n_slot0 + n_slot1;

  // Q rows, loaded now into registers so that the loads overlap barrier set-up and TMEM
  // allocation; they are stored to shared memory after the block barrier.  Two row groups:
  // group g loads its 128 rows, all 16 chunks of 16 bytes; one row group: group g loads
  // head-dim half g of the 128 rows.  Rows past R are zero (their scores are 0 and their
  // output unused).
  uint4 qv[16];
  if (warp >= 4) {
    if (one_call) asm volatile("griddepcontrol.wait;" ::: "memory");
    const int wg = (warp - 4) >> 2, tq = (int)threadIdx.x - 128 - 128 * wg;
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      qv[i] = make_uint4(0u, 0u, 0u, 0u);
      if (!dual && i >= 8) continue;
      const int k = tq + 128 * i;
      const int r = dual ? (k >> 4) : (k >> 3);
      const int c = dual ? (k & 15) : (8 * wg + (k & 7));
      const int qrow = row0 + (dual ? 128 * wg : 0) + r;
      if (qrow < R) {
        const int el = qrow / p.group;
        const int gh = qrow - el * p.group;
        qv[i] = __ldg(reinterpret_cast<const uint4*>(
            q + ((size_t)(it.first_event + el) * p.h_q + kvh * p.group + gh) * kD + 8 * c));
      }
    }
  }

  auto load_k = [&](int t) {
    const int s = t % kKS;
    mbar_expect_tx(&bars->kfull[s], kTileBytes);
    const uint32_t dst = sbase + kOffK + (uint32_t)s * kTileBytes;
    tma_load_3d(dst, &tmK, 0, kvh, tok0 + t * kBN, &bars->kfull[s]);
    tma_load_3d(dst + kHalfBytes, &tmK, 64, kvh, tok0 + t * kBN, &bars->kfull[s]);
  };
  auto load_v = [&](int t) {
    const int s = t % VS;
    mbar_expect_tx(&bars->vfull[s], kTileBytes);
    const uint32_t dst = sbase + v_off(s);
    tma_load_3d(dst, &tmV, 0, kvh, tok0 + t * kBN, &bars->vfull[s]);
    tma_load_3d(dst + kHalfBytes, &tmV, 64, kvh, tok0 + t * kBN, &bars->vfull[s]);
  };

  if (threadIdx.x == 0) {
    // The first tile goes out first (its two barriers initialised, then the loads), before
    // the other barriers, TMEM allocation and the block barrier; the producer thread issues
    // the rest once it has landed, so that every CTA's first tile is not queued in DRAM
    // behind the later tiles of all the others.
    mbar_init(&bars->kfull[0], 1);
    mbar_init(&bars->vfull[0], 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmK)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmV)) : "memory");
    if (one_call) asm volatile("griddepcontrol.wait;" ::: "memory");
    if (n_tiles > 0) {
      load_k(0);
      load_v(0);
    }
    for (int s = 0; s < 3; ++s) {
      if (s > 0) {
        mbar_init(&bars->kfull[s], 1);
        mbar_init(&bars->vfull[s], 1);
      }
      mbar_init(&bars->kfree[s], 1);
      mbar_init(&bars->vfree[s], 1);
    }
    for (int g = 0; g < 2; ++g) {
      mbar_init(&bars->sfull[g], 1);
      mbar_init(&bars->plo[g], 4);  // one arrival per softmax warp of the slot
      mbar_init(&bars->phi[g], 4);
      mbar_init(&bars->pvlo[g], 1);
      mbar_init(&bars->pvdone[g], 1);
    }
    mbar_init(&bars->drain_s, 1);
    mbar_init(&bars->drain_pv, 1);
    mbar_init(&bars->qready, 8);
    mbar_init(&bars->tdone, 8);
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
  // The branch/merge grid after this one may start its prologue now; it waits for this
  // grid's completion before it reads partials.
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const uint32_t tmem = bars->tmem_base;

  if (warp < 4) {
    if (warp == 0) {
      // ------------------------------------------------------------ TMA producer
      if (lane == 0) {
        // K tile t reuses the stage of tile t - 3 once its S MMAs have completed, V tile t the
        // stage of tile t - VS once its P.V MMAs have; issued in the order the MMAs use them
        // (V(t), then K(t + 1)).
        int issued_k = min(1, n_tiles), issued_v = min(1, n_tiles);
        bool ok = n_tiles <= 1 || dwait(&bars->kfull[0], 0u, bars, p.header, 1);
        for (int t = 1; t < n_tiles && ok; ++t) {
          if (t >= kKS) ok = dwait(&bars->kfree[t % kKS], (uint32_t)((t / kKS - 1) & 1), bars, p.header, 1);
          if (!ok) break;
          load_k(t);
          issued_k = t + 1;
          if (t >= VS) ok = dwait(&bars->vfree[t % VS], (uint32_t)((t / VS - 1) & 1), bars, p.header, 2);
          if (!ok) break;
          load_v(t);
          issued_v = t + 1;
        }
        if (!ok) {
          // the loads already issued must land before the CTA leaves
          for (int t = max(0, issued_k - kKS); t < issued_k; ++t)
            drain_wait(&bars->kfull[t % kKS], (uint32_t)((t / kKS) & 1));
          for (int t = max(0, issued_v - VS); t < issued_v; ++t)
            drain_wait(&bars->vfull[t % VS], (uint32_t)((t / VS) & 1));
        }
      }
      __syncwarp();
      if (!p.causal) prefetch_branch_tasks(p, q, kpool, vpool, lane);
    } else if (warp == 1 || warp == 2) {
      // ------------------------------------------------------------ MMA issuers
      // Two threads feed the tensor pipe, so that one's waits do not hold back the other's
      // MMAs: warp 1 issues S = Q K^T, warp 2 (after allocating TMEM) O += P V.  A commit
      // tracks only its own thread's MMAs, so each has its own completion barriers.
      if (lane == 0) {
        bool ok = true;
        if (warp == 1) {
          // Descriptors are built once; a K-step moves the start address, i.e. adds
          // (byte offset >> 4) to the low field (no carry: addresses stay below 256 KB).
          const uint64_t dQ0 = sdesc(sbase + kOffQ0, 16, 1024);
          const uint64_t dQ1 = sdesc(sbase + kOffQ1, 16, 1024);
          const uint64_t dK = sdesc(sbase + kOffK, 16, 1024);
          // S_g(k): waits for the K tile and for the P.V of the slot's previous tile (its
          // P lives in the S buffer this MMA overwrites).  The K stage is released by the
          // commit after the last S that reads it.
          ok = dwait(&bars->qready, 0u, bars, p.header, 11);
          for (int i = 0; i < n_seq && ok; ++i) {
            const int g = i & 1, k = i >> 1, t = dual ? k : i, s = t % kKS;
            if (!dual || g == 0) ok = dwait(&bars->kfull[s], (uint32_t)((t / kKS) & 1), bars, p.header, 3);
            if (ok && k > 0) ok = dwait(&bars->pvdone[g], (uint32_t)((k - 1) & 1), bars, p.header, 6);
            if (!ok) break;
            fence_after();
            const uint64_t qd = (dual && g == 1) ? dQ1 : dQ0;
            const uint64_t kb = dK + ((uint32_t)s * kTileBytes >> 4);
#pragma unroll
            for (int kk = 0; kk < kD / 16; ++kk) {
              const uint32_t off = (uint32_t)(kk >> 2) * kQHalfBytes + (uint32_t)(kk & 3) * 32;
              mma_ss(tmem + 128u * g, qd + (off >> 4), kb + (off >> 4), kIdescS, kk > 0 ? 1u : 0u);
            }
            mma_commit(&bars->sfull[g]);
            if (!dual || g == 1) mma_commit(&bars->kfree[s]);
          }
          mma_commit(&bars->drain_s);
          drain_wait(&bars->drain_s, 0u);
        } else {
          // O_g += P_g(k) V, in two halves of 64 tokens: each waits for the slot's P of that
          // half, so the first runs while the softmax still works on the second.  V tile,
          // N(=head-dim)-major: 16 tokens per K-step (2048 bytes), the second 64-column
          // half at +kHalfBytes (leading byte offset), 8-row groups 1024 apart.
          for (int i = 0; i < n_seq && ok; ++i) {
            const int g = i & 1, k = i >> 1, t = dual ? k : i, s = t % VS;
            if (!dual || g == 0) ok = dwait(&bars->vfull[s], (uint32_t)((t / VS) & 1), bars, p.header, 4);
            const uint64_t vb = sdesc(sbase + v_off(s), kHalfBytes, 1024);
#pragma unroll
            for (int hh = 0; hh < 2; ++hh) {
              if (ok) ok = dwait(hh ? &bars->phi[g] : &bars->plo[g], (uint32_t)(k & 1), bars, p.header, 5);
              if (!ok) break;
              fence_after();
#pragma unroll
              for (int kk = 4 * hh; kk < 4 * hh + 4; ++kk)
                mma_ts(tmem + kColO + 128u * g, tmem + 128u * g + kk * 8, vb + ((uint32_t)kk * 2048 >> 4), kIdescPV,
                       (k > 0 || kk > 0) ? 1u : 0u);
              if (hh == 0) mma_commit(&bars->pvlo[g]);
            }
            if (!ok) break;
            mma_commit(&bars->pvdone[g]);
            if (!dual || g == 1) mma_commit(&bars->vfree[s]);
          }
          mma_commit(&bars->drain_pv);
          drain_wait(&bars->drain_pv, 0u);
        }
      }
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ softmax
    const int wg = (warp - 4) >> 2;            // slot
    const int q4 = warp & 3;                   // TMEM lanes 32*q4 .. +31
    // Q rows (loaded in the prologue) into the 128-byte-swizzled K-major layout the MMA
    // reads: row r, 16-byte chunk c (of 16) at (c / 8) * 16K + r * 128 + ((c % 8) ^ (r % 8)) * 16.
    {
      const int tq = (int)threadIdx.x - 128 - 128 * wg;
      const uint32_t qbase = (dual && wg == 1) ? kOffQ1 : kOffQ0;
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        if (!dual && i >= 8) continue;
        const int k = tq + 128 * i;
        const int r = dual ? (k >> 4) : (k >> 3);
        const int c = dual ? (k & 15) : (8 * wg + (k & 7));
        *reinterpret_cast<uint4*>(smem + qbase + (c >> 3) * kQHalfBytes + r * 128 + (((c & 7) ^ (r & 7)) << 4)) = qv[i];
      }
    }
    if (ROPE) {
      // Rotation in place: element d < 64 pairs with d + 64, i.e. chunk cc of half 0 with
      // chunk cc of half 1 of the same row (with one row group the two halves were stored
      // by different groups, so all 256 threads meet first and then split the pairs).
      asm volatile("bar.sync 1, 256;" ::: "memory");
      const int t256 = (int)threadIdx.x - 128;
      const int n_pairs = (dual ? 256 : 128) * 8;
      for (int k = t256; k < n_pairs; k += 256) {
        const int sl = k >> 10, rr = (k & 1023) >> 3, cc = k & 7;
        const int qrow = row0 + 128 * sl + rr;
        if (qrow >= R) continue;
        const float* cs = p.rope_cs + (size_t)plan_events(p)[it.first_event + qrow / p.group].pos * kD;
        const uint32_t base = sl ? kOffQ1 : kOffQ0;
        uint4* lo = reinterpret_cast<uint4*>(smem + base + rr * 128 + ((cc ^ (rr & 7)) << 4));
        uint4* hi = reinterpret_cast<uint4*>(smem + base + kQHalfBytes + rr * 128 + ((cc ^ (rr & 7)) << 4));
        const uint4 a = *lo, b = *hi;
        const float4 c0 = *reinterpret_cast<const float4*>(cs + 8 * cc);
        const float4 c1 = *reinterpret_cast<const float4*>(cs + 8 * cc + 4);
        const float4 s0 = *reinterpret_cast<const float4*>(cs + 64 + 8 * cc);
        const float4 s1 = *reinterpret_cast<const float4*>(cs + 64 + 8 * cc + 4);
        const float cv[8] = {c0.x, c0.y, c0.z, c0.w, c1.x, c1.y, c1.z, c1.w};
        const float sv[8] = {s0.x, s0.y, s0.z, s0.w, s1.x, s1.y, s1.z, s1.w};
        const uint32_t av[4] = {a.x, a.y, a.z, a.w}, bv[4] = {b.x, b.y, b.z, b.w};
        uint32_t ol[4], oh[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const float2 x = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&av[j]));
          const float2 y = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&bv[j]));
          ol[j] = pack_bf16(rope_one(x.x, y.x, cv[2 * j], sv[2 * j], true),
                            rope_one(x.y, y.y, cv[2 * j + 1], sv[2 * j + 1], true));
          oh[j] = pack_bf16(rope_one(y.x, x.x, cv[2 * j], sv[2 * j], false),
                            rope_one(y.y, x.y, cv[2 * j + 1], sv[2 * j + 1], false));
        }
        *lo = make_uint4(ol[0], ol[1], ol[2], ol[3]);
        *hi = make_uint4(oh[0], oh[1], oh[2], oh[3]);
      }
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    __syncwarp();
    if (lane == 0) mbar_arrive(&bars->qready);

    const int row = 32 * q4 + lane;                     // TMEM lane: row within the slot
    const int srow = (dual ? 128 * wg : 0) + row;       // row within the CTA
    const int grow = row0 + srow;                       // row within the item
    const bool warp_active = row0 + (dual ? 128 * wg : 0) + 32 * q4 < R;
    const uint32_t tl = tmem + ((uint32_t)(32 * q4) << 16);
    const uint32_t cS = 128u * (uint32_t)wg, cO = kColO + 128u * (uint32_t)wg;
    const int n_mine = wg ? n_slot1 : n_slot0;
    const float sl2 = p.scale_log2;
    float m_run = -__builtin_huge_valf(), l_run = 0.f;
    bool ok = true;
    // self G-token mask: the video's planning tokens G^1..G^K (prefix-relative [g_lo, g_hi))
    // and this row's own one
    int g_lo = 0, g_hi = 0, g_own = -1;
    if (GSELF) {
      const PadVideoDesc vdg = plan_videos(p)[plan_events(p)[it.first_event].video];
      if (vdg.n_planning > 0) {
        g_lo = vdg.prefix_len - 1 - vdg.n_planning;
        g_hi = vdg.prefix_len - 1;
        if (grow < R) g_own = g_lo + plan_events(p)[it.first_event + grow / p.group].gidx;
      }
    }
    for (int k = 0; k < n_mine; ++k) {
      const int t = dual ? k : 2 * k + wg;
      ok = dwait(&bars->sfull[wg], (uint32_t)(k & 1), bars, p.header, 8);
      ok = __all_sync(0xffffffffu, ok);  // tcgen05.ld/st below are warp-collective
      if (!ok) break;
      fence_after();
      if (warp_active) {
        // columns to mask: past the split's end, or (GSELF) hidden planning tokens of this
        // row's event; the path is chosen per warp (tcgen05.ld/st are warp-collective)
        const int valid = min(kBN, ntok - t * kBN);
        uint64_t keep0 = low_bits(valid), keep1 = low_bits(valid - 64);
        bool masked = valid < kBN;
        if (GSELF) {
          const int t0 = it.tok_begin + t * kBN;
          if (g_lo < g_hi && t0 < g_hi && t0 + kBN > g_lo) {
            const GMask gm{g_lo, g_hi, g_own};
            keep0 = keep_bits(valid, gm, t0);
            keep1 = keep_bits(valid - 64, gm, t0 + 64);
          }
          masked = __any_sync(0xffffffffu, (keep0 & keep1) != ~0ull);
        }
        // Half rows in turn: P of a half is computed with the running maximum in the same
        // pass that finds the half's maximum; only when that grows past the running one by
        // more than the lazy bound (always on the first half of the slot's first tile) is
        // the half redone from its registers, after O and l are scaled down to the new
        // maximum.  P goes over the first 64 columns of the S buffer (token n in column
        // n / 2), whose S values are read by then; the first half's P is released to the
        // P.V issuer as soon as it is written.
#pragma unroll 1
        for (int hh = 0; hh < 2; ++hh) {
          uint32_t h[2][32], pk[32];
          tmem_ld32(tl + cS + 64 * hh, h[0]);
          tmem_ld32(tl + cS + 64 * hh + 32, h[1]);
          tmem_wait_ld_dep(h[0]);
          tmem_wait_ld_dep(h[1]);
          if (masked) mask_half(h, hh ? keep1 : keep0);
          float sum = 0.f;
#pragma unroll 1
          for (int pass = 0; pass < 2; ++pass) {
            // a row with every key so far hidden keeps m = -inf; its exponent base is 0
            const float mu = m_run == -__builtin_huge_valf() ? 0.f : m_run;
            float mx;
            sum = half_exp(h, sl2, mu, pk, &mx);
            const float m_new = fmaxf(m_run, mx * sl2);
            const bool grow = m_new > m_run + kLazyRescale;
            if (pass == 1 || !__any_sync(0xffffffffu, grow)) break;
            // rescale to the new maximum: O and l.  O holds P.V of the slot's earlier tiles
            // once the previous one has completed, and (second half) also that of this
            // tile's first half once its P.V has completed
            if (k > 0 || hh == 1) {
              ok = hh ? dwait(&bars->pvlo[wg], (uint32_t)(k & 1), bars, p.header, 9)
                      : dwait(&bars->pvdone[wg], (uint32_t)((k - 1) & 1), bars, p.header, 9);
              ok = __all_sync(0xffffffffu, ok);
              if (!ok) break;
              fence_after();
            }
            const float alpha = grow ? ex2(m_run - m_new) : 1.f;
            uint32_t r[32];
            if (k > 0 || hh == 1) {
#pragma unroll 1
              for (int c = 0; c < 4; ++c) {
                tmem_ld32(tl + cO + 32 * c, r);
                tmem_wait_ld_dep(r);
#pragma unroll
                for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * alpha);
                tmem_st32(tl + cO + 32 * c, r);
              }
            }
            tmem_wait_st();
            l_run *= alpha;
            if (grow) m_run = m_new;
          }
          if (!ok) break;
          l_run += sum;
          tmem_st32(tl + cS + 32 * hh, pk);
          if (hh == 0) {
            // the first half's P is in place: its P.V may start
            tmem_wait_st();
            fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&bars->plo[wg]);
          }
        }
        if (!ok) break;
        tmem_wait_st();
      } else {
        if (lane == 0) mbar_arrive(&bars->plo[wg]);
      }
      fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars->phi[wg]);
    }
    // The slot's O is final once its last P.V has completed (which, issued by one thread,
    // implies every earlier P.V: after slot 1's the V stages are idle); the K stages are
    // idle once the S issuer's last MMA has completed.  They hold the O rows for the
    // write-out.
    if (ok && n_mine > 0) ok = dwait(&bars->pvdone[wg], (uint32_t)((n_mine - 1) & 1), bars, p.header, 10);
    // With two row groups, slot 0 stages into the K stages: the S issuer's last MMA
    // (slot 1's, issued after slot 0's last S, which is all this group has seen complete)
    // must have finished reading them.
    if (ok && dual && wg == 0) ok = dwait(&bars->drain_s, 0u, bars, p.header, 14);
    ok = __all_sync(0xffffffffu, ok);
    uint32_t r[32];
    if (dual) {
      // two row groups: each writes its own rows' partial state
      uint8_t* stg = smem + (wg ? kOffV : kOffK);
      if (ok && warp_active) {
        fence_after();
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          tmem_ld32(tl + cO + 32 * c, r);
          tmem_wait_ld_dep(r);
#pragma unroll
          for (int j = 0; j < 8; ++j)
            *reinterpret_cast<uint4*>(stg + stage_off(row, 8 * c + j)) =
                make_uint4(r[4 * j], r[4 * j + 1], r[4 * j + 2], r[4 * j + 3]);
        }
        if (grow < R) p.part_ml[(int64_t)it.part_row0 + grow] = make_float2(m_run, l_run);
      }
      fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars->tdone);
      asm volatile("bar.sync %0, 128;" ::"r"(2 + wg) : "memory");
      if (ok) {
        const int nrows = min(128, R - row0 - 128 * wg);
        for (int rr = q4; rr < nrows; rr += 4) {
          const uint4 v = *reinterpret_cast<const uint4*>(stg + stage_off(rr, lane));
          *reinterpret_cast<uint4*>(p.part_o + ((int64_t)it.part_row0 + row0 + 128 * wg + rr) * kD + 4 * lane) = v;
        }
      }
    } else {
      // one row group: merge the two parities' states, O = 2^(m_0 - M) O_0 + 2^(m_1 - M) O_1;
      // group g combines head-dim columns 64g .. 64g+63
      float2* xs = reinterpret_cast<float2*>(smem + kOffX);  // [slot][row] (m, l)
      xs[wg * 128 + row] = make_float2(m_run, l_run);
      asm volatile("bar.sync 1, 256;" ::: "memory");
      uint8_t* stg = smem + kOffK;
      if (ok && warp_active) {
        const float2 a = xs[row], b = xs[128 + row];
        const float M = fmaxf(a.x, b.x);
        const float Mu = M == -__builtin_huge_valf() ? 0.f : M;
        const float fa = ex2(a.x - Mu), fb = ex2(b.x - Mu);
        fence_after();
#pragma unroll
        for (int c = 0; c < 2; ++c) {
          const uint32_t col = 64u * (uint32_t)wg + 32u * (uint32_t)c;
          uint32_t rb[32];
          tmem_ld32(tl + kColO + col, r);
          if (n_slot1 > 0) tmem_ld32(tl + kColO + 128 + col, rb);
          tmem_wait_ld_dep(r);
          if (n_slot1 > 0) {
            tmem_wait_ld_dep(rb);
#pragma unroll
            for (int i = 0; i < 32; ++i)
              r[i] = __float_as_uint(__uint_as_float(r[i]) * fa + __uint_as_float(rb[i]) * fb);
          } else {
#pragma unroll
            for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * fa);
          }
#pragma unroll
          for (int j = 0; j < 8; ++j)
            *reinterpret_cast<uint4*>(stg + stage_off(row, (int)(col >> 2) + j)) =
                make_uint4(r[4 * j], r[4 * j + 1], r[4 * j + 2], r[4 * j + 3]);
        }
        if (wg == 0 && grow < R) p.part_ml[(int64_t)it.part_row0 + grow] = make_float2(M, a.y * fa + b.y * fb);
      }
      fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars->tdone);
      asm volatile("bar.sync 1, 256;" ::: "memory");
      if (ok) {
        for (int rr = warp - 4; rr < rows; rr += 8) {
          const uint4 v = *reinterpret_cast<const uint4*>(stg + stage_off(rr, lane));
          *reinterpret_cast<uint4*>(p.part_o + ((int64_t)it.part_row0 + row0 + rr) * kD + 4 * lane) = v;
        }
      }
    }
    __syncwarp();
  }

  __syncwarp();
  fence_before();
  // This grid may run alongside the append kernel before it (it reads nothing that kernel
  // writes); waiting for it here makes the completion of this grid imply the completion
  // of the append, which the branch/merge pass after it relies on.
  if (threadIdx.x == 0) asm volatile("griddepcontrol.wait;" ::: "memory");
  __syncthreads();
  if (warp == 2) {
    // the softmax warps' own arrivals order their last TMEM reads before the deallocation
    drain_wait(&bars->tdone, 0u);
    fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols)
                 : "memory");
  }
}

}  // namespace

cudaError_t launch_prefix_dual(const KParams& p, int max_rows, const void* q, const void* kp, const void* vp,
                               int64_t total_prefix_tokens, const void* k_pool, const void* v_pool, bool pdl,
                               cudaStream_t s) {
  if (p.n_items == 0) return cudaSuccess;
  if (p.head_dim != kD || total_prefix_tokens <= 0 || total_prefix_tokens > (int64_t)INT32_MAX || p.fused)
    return cudaErrorInvalidValue;
  int dev = 0;
  cudaGetDevice(&dev);
  CUtensorMap mk, mv;
  if (!prefix_tensor_maps(kp, vp, p.h_kv, total_prefix_tokens, dev, &mk, &mv)) return cudaErrorInvalidValue;
  static bool configured[64] = {};
  if (dev >= 0 && dev < 64 && !configured[dev]) {
    for (auto fn : {prefix_dual_kernel<false, false>, prefix_dual_kernel<true, false>, prefix_dual_kernel<false, true>,
                    prefix_dual_kernel<true, true>}) {
      cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
      if (e != cudaSuccess) return e;
    }
    configured[dev] = true;
  }
  const int n_groups = (max_rows + 255) / 256;
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
  auto fn = p.rope_cs != nullptr ? (p.g_self ? prefix_dual_kernel<true, true> : prefix_dual_kernel<true, false>)
                                 : (p.g_self ? prefix_dual_kernel<false, true> : prefix_dual_kernel<false, false>);
  return cudaLaunchKernelEx(&cfg, fn, p, static_cast<const __nv_bfloat16*>(q), n_groups, mk, mv,
                            static_cast<const __nv_bfloat16*>(k_pool), static_cast<const __nv_bfloat16*>(v_pool));
}

}  // namespace pad
