// Internal declarations shared by the host planner (pad_api.cu) and the kernels.
// The device-side plan is a flat block at the start of the caller's workspace:
//
//   [0, 256)            PadDevHeader (status word, tagged with the plan's generation)
//   videos              PadVideoDesc[n_videos]
//   events              PadEventDesc[n_events]
//   items               PadWorkItem[n_work_items]       (prefix split-KV work list)
//   -- end of the plan image --
//   part_ml             float2[partial_rows]            (m in log2 units, l)
//   part_o              float[partial_rows * head_dim]  (unnormalised O)
//
// Partial row of (video b, kv-head h, split s, row r) with r = e_local * G + g:
//   part_base[b] + (h * n_splits[b] + s) * R_b + r,   R_b = n_events[b] * G.
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "../../include/pad.h"

namespace pad {

constexpr int kSplitGranule = 128;   // prefix splits are multiples of this many tokens
constexpr int kMaxGroup = 16;        // G = h_q / h_kv supported by the kernels

// Status word of a workspace.  Each plan carries a fresh 56-bit generation; kernels record
// the first error of their generation as (generation << 8) | pad_status, and a word that
// carries another generation counts as clear, so nothing resets it between steps.
struct PadDevHeader {
  unsigned long long word;
  int32_t info[3];     // kernel-specific detail of that error (e.g. event, page)
  int32_t pad[59];
};
static_assert(sizeof(PadDevHeader) == 256, "header is 256 bytes");

#ifdef __CUDACC__
__device__ __forceinline__ void pad_set_error(PadDevHeader* h, uint64_t gen, int code, int a, int b,
                                              int c) {
  const unsigned long long want = ((unsigned long long)gen << 8) | (unsigned)code;
  unsigned long long cur = *reinterpret_cast<volatile unsigned long long*>(&h->word);
  while ((cur >> 8) != gen || (cur & 0xffull) == 0) {
    const unsigned long long prev = atomicCAS(&h->word, cur, want);
    if (prev == cur) {
      h->info[0] = a;
      h->info[1] = b;
      h->info[2] = c;
      return;
    }
    cur = prev;
  }
}
#endif

struct PadVideoDesc {
  int64_t prefix_off;   // first token of the prefix in k_prefix / v_prefix
  int32_t prefix_len;
  int32_t first_event;
  int32_t n_events;
  int16_t n_splits;     // prefix splits per kv-head (0 if prefix_len == 0 or no events)
  int16_t n_planning;   // K of the "self G-token only" mask (its G^1..G^K, S end the
                        // prefix), 0 = every event sees every prefix token
  int32_t part_base;    // first partial row of this video
  int32_t cnt_base;     // first split counter of this video (fused tail; see KParams::counters)
};
static_assert(sizeof(PadVideoDesc) == 32, "video desc is 32 bytes");

struct PadEventDesc {
  int32_t new_page;     // page taken this step, or -1
  int32_t pos;          // position of this step's token (rotary table row; 0 without RoPE)
  uint16_t len;         // private length before this step
  uint16_t video;
  uint16_t local;       // index of the event within its video
  uint16_t gidx;        // its own planning token G^(gidx+1) (self G-token mask only)
};
static_assert(sizeof(PadEventDesc) == 16, "event desc is 16 bytes");

// One prefix split of one (video, kv-head).  It carries copies of the owning video's
// fields so that a CTA can start after a single 32-byte load.
struct PadWorkItem {
  int64_t tok0;         // first token of the split in k_prefix / v_prefix (prefix_off + tok_begin)
  int32_t tok_begin;    // [tok_begin, tok_end) relative to the video's prefix start
  int32_t tok_end;
  int32_t first_event;  // the video's first event and event count
  int32_t n_events;
  int32_t part_row0;    // partial row of (this split, row 0): part_base + (kvh * n_splits + split) * R
  int16_t kvh;
  int16_t split;
};
static_assert(sizeof(PadWorkItem) == 32, "work item is 32 bytes");

constexpr int kParamImageBytes = 8192 - 256;  // descriptor bytes carried in KParams

// Everything a kernel needs, passed by value.
struct KParams {
  int32_t h_q, h_kv, group, head_dim, page_size, max_pages, n_pages;
  int32_t n_videos, n_events, n_items;
  int32_t out_bf16;
  int32_t n_sms;                  // SMs the grid sizes were planned for
  int32_t max_splits;             // largest per-video prefix split count of the batch
  int32_t branch_rows;            // branch keys staged per round: the longest branch's
                                  // len + 1 rounded up to 16, at most 128
  int32_t fused;                  // the tensor-core prefix kernel runs a4 + a5 itself (one
                                  // (event, kv-head) task per CTA after its split)
  int32_t tail_chunk;             // split partials merged per staged chunk in that tail
  int32_t merge_first;            // one-call step whose prefix grid leaves too few SMs for
                                  // the branch/merge CTAs to run beside it: each of them
                                  // waits for it first, then stages the split partials
                                  // while its branch pass runs
  float scale_log2;               // scale * log2(e)
  uint64_t gen;                   // generation of the plan (tags errors in the status word)
  PadDevHeader* header;
  const PadVideoDesc* videos;
  const PadEventDesc* events;
  const PadWorkItem* items;
  float2* part_ml;
  float* part_o;
  int32_t* page_table;
  // Set by the one-call step (pad_decode_step): this step's new K/V rows [n_events, h_kv,
  // head_dim].  Each (event, kv-head) task of a4 then reads its key `len` from here and
  // writes it into the pools itself (a2 folded into a4; no append kernel runs).
  const void* k_new;
  const void* v_new;
  // Rotary table [max_position, head_dim] fp32 (cos | sin halves) when the plan carries
  // positions (pad_plan_set_rope): q and the new key are rotated where they are loaded.
  const float* rope_cs;
  int32_t g_self;                 // "self G-token only" mask: videos with n_planning > 0
  int32_t causal;                 // "causal attention" mask: every branch's stored tokens
                                  // are visible to every branch of the video
  // Whole-sequence prefill on the tensor-core kernel (pad_prefill_attn): a CTA takes
  // pf_tpc query tokens x G heads of one kv-head against its visible key ranges and writes
  // the normalised output; branch b of the sequence starts at token ((int32_t*)img)[b]
  // (b <= pf_nb, entry 0 = pf_S).
  int32_t pf_N, pf_S, pf_nb, pf_tpc;
  void* pf_out;
  float* pf_lse;
  const int32_t* tasks;           // per prefix CTA: its (event * h_kv + kv-head) task, or -1
                                  // (fused tail); with cta_map its (work item << 6) | row group
  int32_t cta_map;                // the tensor-core prefix grid is the n_ctas CTAs of that list
  int32_t n_ctas;
  // Per (video, kv-head, 128-row group): bits 15-0 how many of the video's prefix splits
  // have written their partials, bits 31-16 how many tasks have taken them.  Zeroed by
  // the append kernel of the step; the last task to take a counter zeroes it again, so a
  // plan launched twice without an append in between starts from zero too.
  unsigned int* counters;
  int32_t n_counters;
  // The descriptors themselves when they fit (img_n > 0): carried in the launch's
  // parameter block, so a CTA reads them from the constant bank instead of from the
  // plan's page-locked host image.  Sections start at the img_* byte offsets.
  int32_t img_n;                  // bytes used, 0 = read videos / events / items instead
  int32_t img_videos, img_events, img_items, img_tasks;
  alignas(16) unsigned char img[kParamImageBytes];
};
static_assert(sizeof(KParams) <= 8192, "kernel parameters stay at 8 KB");

#ifdef __CUDACC__
// Kernels take their KParams as a __grid_constant__ parameter, so these point into the
// parameter block itself.
__device__ __forceinline__ const PadVideoDesc* plan_videos(const KParams& p) {
  return p.img_n > 0 ? reinterpret_cast<const PadVideoDesc*>(p.img + p.img_videos) : p.videos;
}
__device__ __forceinline__ const PadEventDesc* plan_events(const KParams& p) {
  return p.img_n > 0 ? reinterpret_cast<const PadEventDesc*>(p.img + p.img_events) : p.events;
}
__device__ __forceinline__ const PadWorkItem* plan_items(const KParams& p) {
  return p.img_n > 0 ? reinterpret_cast<const PadWorkItem*>(p.img + p.img_items) : p.items;
}
__device__ __forceinline__ const int32_t* plan_tasks(const KParams& p) {
  return p.img_n > 0 ? reinterpret_cast<const int32_t*>(p.img + p.img_tasks) : p.tasks;
}

// "Self G-token only" mask (attention ablation of the paper, Tab. 8): a row of event e
// does not see the planning tokens G^1..G^K of its video other than its own; the prefix
// ends with them and S.  Token indices are relative to the video's prefix.
struct GMask {
  int lo, hi, own;  // hidden: lo <= t < hi, t != own (lo == hi: nothing hidden)
};
__device__ __forceinline__ GMask g_mask_of(const KParams& p, const PadVideoDesc& vd, const PadEventDesc& ev) {
  if (!p.g_self || vd.n_planning == 0) return GMask{0, 0, -1};
  const int lo = vd.prefix_len - 1 - vd.n_planning;
  return GMask{lo, vd.prefix_len - 1, lo + ev.gidx};
}
__device__ __forceinline__ bool g_visible(const GMask& g, int t) { return t < g.lo || t >= g.hi || t == g.own; }
// Visible-column bits of the 64 tokens t0 .. t0+63, given the first `valid` are in range.
__device__ __forceinline__ uint64_t keep_bits(int valid, const GMask& g, int t0) {
  uint64_t keep = valid >= 64 ? ~0ull : (valid <= 0 ? 0ull : ((1ull << valid) - 1ull));
  const int a = max(g.lo - t0, 0), b = min(g.hi - t0, 64);
  if (a < b) {
    const uint64_t range = (b >= 64 ? ~0ull : ((1ull << b) - 1ull)) & ~((1ull << a) - 1ull);
    const int o = g.own - t0;
    keep &= ~range | ((o >= 0 && o < 64) ? (1ull << o) : 0ull);
  }
  return keep;
}

// Rotary embedding, rotate-half form (the position rule of Sec. 3.4 decides `cs`, the
// table row of the token's position: cos in columns i < D/2, sin in D/2 + i).  Element
// d < D/2 becomes x_d cos_d - x_{d+D/2} sin_d, element D/2 + i becomes
// x_{D/2+i} cos_i + x_i sin_i; each product and sum is rounded to fp32 (no contraction)
// and the result once to bf16, as an unfused rotation pass would store it.
__device__ __forceinline__ float rope_one(float own, float partner, float c, float s, bool low) {
  return low ? __fsub_rn(__fmul_rn(own, c), __fmul_rn(partner, s))
             : __fadd_rn(__fmul_rn(own, c), __fmul_rn(partner, s));
}
// Elements d0 .. d0+7 (d0 a multiple of 8) of a bf16 row of length D, as packed bf16.
__device__ __forceinline__ uint4 rope_chunk8(const __nv_bfloat16* row, int D, int d0, const float* cs) {
  const int h = D >> 1;
  const bool low = d0 < h;
  const int i0 = low ? d0 : d0 - h;
  const uint4 xa = *reinterpret_cast<const uint4*>(row + d0);
  const uint4 xb = *reinterpret_cast<const uint4*>(row + (low ? d0 + h : i0));
  const float4 c0 = *reinterpret_cast<const float4*>(cs + i0), c1 = *reinterpret_cast<const float4*>(cs + i0 + 4);
  const float4 s0 = *reinterpret_cast<const float4*>(cs + h + i0),
               s1 = *reinterpret_cast<const float4*>(cs + h + i0 + 4);
  const float c[8] = {c0.x, c0.y, c0.z, c0.w, c1.x, c1.y, c1.z, c1.w};
  const float s[8] = {s0.x, s0.y, s0.z, s0.w, s1.x, s1.y, s1.z, s1.w};
  const uint32_t a[4] = {xa.x, xa.y, xa.z, xa.w}, b[4] = {xb.x, xb.y, xb.z, xb.w};
  uint32_t o[4];
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const float2 x = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&a[j]));
    const float2 y = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&b[j]));
    const __nv_bfloat162 r = __floats2bfloat162_rn(rope_one(x.x, y.x, c[2 * j], s[2 * j], low),
                                                   rope_one(x.y, y.y, c[2 * j + 1], s[2 * j + 1], low));
    o[j] = *reinterpret_cast<const uint32_t*>(&r);
  }
  return make_uint4(o[0], o[1], o[2], o[3]);
}
// Elements d, d+1 (d even) as packed bf16.
__device__ __forceinline__ uint32_t rope_pair(const __nv_bfloat16* row, int D, int d, const float* cs) {
  const int h = D >> 1;
  const bool low = d < h;
  const int i0 = low ? d : d - h;
  const float2 x = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(row + d));
  const float2 y = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(row + (low ? d + h : i0)));
  const float2 c = *reinterpret_cast<const float2*>(cs + i0), s = *reinterpret_cast<const float2*>(cs + h + i0);
  const __nv_bfloat162 r = __floats2bfloat162_rn(rope_one(x.x, y.x, c.x, s.x, low), rope_one(x.y, y.y, c.y, s.y, low));
  return *reinterpret_cast<const uint32_t*>(&r);
}
// Element d, widened back to fp32 after the bf16 rounding.
__device__ __forceinline__ float rope_elem(const __nv_bfloat16* row, int D, int d, const float* cs) {
  const int h = D >> 1;
  const bool low = d < h;
  const int i = low ? d : d - h;
  const float v = rope_one(__bfloat162float(row[d]), __bfloat162float(row[low ? d + h : i]), cs[i], cs[h + i], low);
  return __bfloat162float(__float2bfloat16_rn(v));
}
#endif

// Launchers (pad_kernels.cu, pad_prefix_tc.cu).  Return the launch error.
cudaError_t launch_host_in(const void* const* src, void* const* dst, const size_t* bytes, int n, int sms,
                           cudaStream_t s);
cudaError_t launch_append(const KParams& p, const void* k_new, const void* v_new, void* k_pool,
                          void* v_pool, cudaStream_t s);
cudaError_t launch_prefix_simt(const KParams& p, int max_rows, const void* q, const void* kp,
                               const void* vp, cudaStream_t s);
cudaError_t launch_prefix_mma(const KParams& p, int max_rows, const void* q, const void* kp,
                              const void* vp, cudaStream_t s);
// With p.fused the same launch also runs a4 + a5 (k_pool, v_pool, out, lse used).
// Split partials merged per staged chunk by that tail (fits the kernel's shared memory).
int prefix_tc_tail_chunk(int branch_rows, int group, int max_splits);
cudaError_t launch_prefix_tc(const KParams& p, int max_rows, const void* q, const void* kp,
                             const void* vp, int64_t total_prefix_tokens, const void* k_pool,
                             const void* v_pool, void* out, float* lse, bool pdl, cudaStream_t s);
// The prefix pass with two softmax groups per CTA (pad_prefix_dual.cu), head_dim 128, not
// fused: up to 256 rows per CTA.
cudaError_t launch_prefix_dual(const KParams& p, int max_rows, const void* q, const void* kp, const void* vp,
                               int64_t total_prefix_tokens, const void* k_pool, const void* v_pool, bool pdl,
                               cudaStream_t s);
// pdl: launch with programmatic stream serialization (the kernel waits for its
// predecessor with griddepcontrol.wait before it reads anything the predecessor wrote).
// Full-sequence prefill / training forward (pad_prefill.cu).
cudaError_t launch_prefill(int32_t n_tokens, int32_t prefix_len, int32_t n_branches, const int32_t* branch_len,
                           int32_t h_q, int32_t h_kv, int32_t head_dim, float scale, int32_t out_bf16, const void* q,
                           const void* k, const void* v, void* out, float* lse, cudaStream_t s);
// The same on the tensor-core kernel (pad_prefix_tc.cu), head_dim 128; device errors go to
// the library's prefill status word (prefill_header), tagged with `gen`.
cudaError_t launch_prefill_tc(int32_t n_tokens, int32_t prefix_len, int32_t n_branches, const int32_t* branch_len,
                              int32_t h_q, int32_t h_kv, float scale, int32_t out_bf16, uint64_t gen, const void* q,
                              const void* k, const void* v, void* out, float* lse, cudaStream_t s);
cudaError_t prefill_header(PadDevHeader** out);
// Grounding readout (pad_ground.cu).  cudaErrorInvalidValue for bad segment offsets.
cudaError_t launch_ground_pool(const void* f_proj, int64_t n_tokens, int32_t d, const int32_t* offsets,
                               int32_t n_segments, float* seg_sum, cudaStream_t s);
cudaError_t launch_ground_score(const void* g_proj, int32_t n_events, const float* seg_sum, int32_t n_segments,
                                int32_t d, float frac, float* scores, uint8_t* salient, int32_t* interval,
                                cudaStream_t s);
cudaError_t launch_attn_aggregate(const void* x, int64_t n_tokens, int32_t d, const float* attn,
                                  const int32_t* offsets, int32_t n_segments, const int32_t* interval,
                                  int32_t n_events, const void* g_emb, float* seg_ws, float* out, cudaStream_t s);
size_t attn_aggregate_ws_floats(int64_t n_tokens, int32_t n_segments, int32_t d);
cudaError_t launch_branch_merge(const KParams& p, const void* q, const void* k_pool,
                                const void* v_pool, void* out, float* lse, bool pdl, cudaStream_t s);

}  // namespace pad
