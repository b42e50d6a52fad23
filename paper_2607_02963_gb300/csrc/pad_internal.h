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
  int32_t n_splits;     // prefix splits per kv-head (0 if prefix_len == 0 or no events)
  int32_t part_base;    // first partial row of this video
  int32_t cnt_base;     // first split counter of this video (fused tail; see KParams::counters)
};
static_assert(sizeof(PadVideoDesc) == 32, "video desc is 32 bytes");

struct PadEventDesc {
  int32_t video;
  int32_t len;          // private length before this step
  int32_t new_page;     // page taken this step, or -1
  int32_t local;        // index of the event within its video
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
  const int32_t* tasks;           // per prefix CTA: its (event * h_kv + kv-head) task, or -1
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
#endif

// Launchers (pad_kernels.cu, pad_prefix_tc.cu).  Return the launch error.
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
// pdl: launch with programmatic stream serialization (the kernel waits for its
// predecessor with griddepcontrol.wait before it reads anything the predecessor wrote).
cudaError_t launch_branch_merge(const KParams& p, const void* q, const void* k_pool,
                                const void* v_pool, void* out, float* lse, bool pdl, cudaStream_t s);

}  // namespace pad
