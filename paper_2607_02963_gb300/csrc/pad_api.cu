// C ABI of libpad: argument validation, page-pool bookkeeping, the split-KV
// planner, workspace layout, and the launch sequence of one decode step.
#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <atomic>
#include <chrono>
#include <deque>
#include <mutex>
#include <queue>
#include <random>
#include <string>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "pad_internal.h"

using namespace pad;

namespace {
// A named NVTX range around each call of the C ABI that does device work or plans it, so
// that a profiler's timeline shows plan / append / attention / step (no cost without one).
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};


thread_local std::string g_last_error;

pad_status fail(pad_status st, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return st;
}

pad_status cuda_fail(cudaError_t e, const char* what) {
  return fail(PAD_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

constexpr int kDefaultSms = 152;
constexpr int kPrefixFlags = PAD_FLAG_PREFIX_SIMT | PAD_FLAG_PREFIX_MMA | PAD_FLAG_PREFIX_TC | PAD_FLAG_PREFIX_DUAL;

int query_num_sms() {
  static int cache[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
    cudaGetLastError();
    return kDefaultSms;
  }
  if (cache[dev] == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) {
      cudaGetLastError();
      n = kDefaultSms;
    }
    cache[dev] = n;
  }
  return cache[dev];
}

pad_status check_problem(const pad_problem* prob) {
  if (!prob) return fail(PAD_ERR_INVALID_ARG, "problem is NULL");
  if (prob->h_q <= 0 || prob->h_kv <= 0 || prob->h_q % prob->h_kv != 0)
    return fail(PAD_ERR_INVALID_ARG, "h_q=%d must be a positive multiple of h_kv=%d", prob->h_q,
                prob->h_kv);
  const int G = prob->h_q / prob->h_kv;
  if (G > kMaxGroup)
    return fail(PAD_ERR_UNSUPPORTED, "group size h_q/h_kv=%d exceeds %d", G, kMaxGroup);
  if (prob->head_dim != 64 && prob->head_dim != 128)
    return fail(PAD_ERR_UNSUPPORTED, "head_dim=%d (supported: 64, 128)", prob->head_dim);
  const int ps = prob->page_size;
  if (ps != 4 && ps != 8 && ps != 16 && ps != 32 && ps != 64)
    return fail(PAD_ERR_UNSUPPORTED, "page_size=%d (supported: 4, 8, 16, 32, 64)", ps);
  if (!(prob->scale > 0.f) || !std::isfinite(prob->scale))
    return fail(PAD_ERR_INVALID_ARG, "scale must be finite and > 0");
  if (prob->out_dtype != 0 && prob->out_dtype != 1)
    return fail(PAD_ERR_INVALID_ARG, "out_dtype=%d (0 = fp32, 1 = bf16)", prob->out_dtype);
  if (prob->num_sms < 0) return fail(PAD_ERR_INVALID_ARG, "num_sms < 0");
  const int known = PAD_FLAG_PREFIX_SIMT | PAD_FLAG_PREFIX_MMA | PAD_FLAG_PREFIX_TC | PAD_FLAG_PREFIX_DUAL |
                    PAD_FLAG_FUSED_MERGE;
  if (prob->flags & ~known) return fail(PAD_ERR_INVALID_ARG, "unknown flags 0x%x", prob->flags);
  const int f = prob->flags & kPrefixFlags;
  if (f && (f & (f - 1))) return fail(PAD_ERR_INVALID_ARG, "at most one PAD_FLAG_PREFIX_* flag");
  return PAD_OK;
}

// Split-KV decomposition and workspace layout of a batch.
struct Layout {
  int group = 1;
  int n_sms = kDefaultSms;
  int split_len = kSplitGranule;
  int max_rows = 0;
  int prefix_kernel = 0;
  std::vector<int32_t> ev_first, ev_count, n_splits, part_base;
  std::vector<int64_t> vsplit;  // prefix tokens per split, per video
  bool longest_first = false;   // CTA list ordered by descending split length
  int64_t n_items = 0;
  int64_t partial_rows = 0;
  // fused tail of the tensor-core path: per prefix CTA its (event * h_kv + kv-head) task or
  // -1, and per (video, kv-head, row group) a split counter
  bool fused = false;
  // Without the fused tail, the tensor-core kernels take their CTAs from a list of
  // (work item, row group) pairs, (item << 6) | group, kept in cta_task: a video with fewer
  // rows than the batch's largest gets no idle CTAs.
  bool cta_map = false;
  int64_t n_ctas = 0;
  // The branch/merge CTAs of a one-call step wait for the prefix grid before their branch
  // pass (see KParams::merge_first).
  bool merge_first = false;
  std::vector<int32_t> cta_task, cnt_base;
  int64_t n_counters = 0;
  size_t off_videos = 0, off_events = 0, off_items = 0, off_tasks = 0, upload_bytes = 0;
  size_t off_ml = 0, off_o = 0, off_cnt = 0, total_bytes = 0;
};

pad_status compute_layout(const pad_problem* prob, int32_t n_videos, const int32_t* prefix_len,
                          int32_t n_events, const int32_t* event_video, int n_sms, Layout* L) {
  if (n_videos < 0 || n_events < 0) return fail(PAD_ERR_INVALID_ARG, "negative batch size");
  if (n_videos > 0 && !prefix_len) return fail(PAD_ERR_INVALID_ARG, "prefix_len is NULL");
  if (n_events > 0 && !event_video) return fail(PAD_ERR_INVALID_ARG, "event_video is NULL");
  if (n_events > 0 && n_videos == 0) return fail(PAD_ERR_INVALID_ARG, "events without videos");
  if (n_videos > 65535) return fail(PAD_ERR_UNSUPPORTED, "at most 65535 videos per step; got %d", n_videos);
  L->group = prob->h_q / prob->h_kv;
  L->n_sms = n_sms;
  L->ev_first.assign(n_videos, 0);
  L->ev_count.assign(n_videos, 0);
  L->n_splits.assign(n_videos, 0);
  L->part_base.assign(n_videos, 0);
  for (int b = 0; b < n_videos; ++b)
    if (prefix_len[b] < 0) return fail(PAD_ERR_INVALID_ARG, "prefix_len[%d]=%d < 0", b, prefix_len[b]);
  int prev = 0;
  for (int e = 0; e < n_events; ++e) {
    const int v = event_video[e];
    if (v < 0 || v >= n_videos)
      return fail(PAD_ERR_INVALID_ARG, "event_video[%d]=%d outside [0, %d)", e, v, n_videos);
    if (v < prev) return fail(PAD_ERR_INVALID_ARG, "event_video must be non-decreasing (event %d)", e);
    if (L->ev_count[v] == 0) L->ev_first[v] = e;
    L->ev_count[v]++;
    prev = v;
  }
  int max_rows = 0;
  for (int b = 0; b < n_videos; ++b) {
    if (L->ev_count[b] > 65535)
      return fail(PAD_ERR_UNSUPPORTED, "at most 65535 events per video; video %d has %d", b, L->ev_count[b]);
    if (L->ev_count[b] > 0) max_rows = std::max(max_rows, L->ev_count[b] * L->group);
  }
  L->max_rows = max_rows;

  // Prefix kernel: forced by a flag, else the tensor-core path for head_dim 128 and the
  // warp-level paths for head_dim 64 (mma.sync above 8 rows, warp-shuffle below).
  int kern = prob->flags & kPrefixFlags;
  if (kern == 0) {
    if (prob->head_dim == 128)
      kern = PAD_FLAG_PREFIX_TC;
    else
      kern = (max_rows <= 8) ? PAD_FLAG_PREFIX_SIMT : PAD_FLAG_PREFIX_MMA;
  }
  if (kern == PAD_FLAG_PREFIX_SIMT && max_rows > 16)
    return fail(PAD_ERR_UNSUPPORTED, "SIMT prefix path takes at most 16 rows per (video, kv-head); got %d",
                max_rows);
  if ((kern == PAD_FLAG_PREFIX_TC || kern == PAD_FLAG_PREFIX_DUAL) && prob->head_dim != 128)
    return fail(PAD_ERR_UNSUPPORTED, "tcgen05 prefix path takes head_dim 128; got %d", prob->head_dim);
  L->prefix_kernel = kern;

  // Split length: a multiple of kSplitGranule tokens sized so that the prefix work
  // (token-heads, times the 128-row groups each item occupies on the tensor-core path)
  // spreads over one wave of SMs.  The tensor-core kernel runs one CTA per SM, so its
  // split is grown until items x row groups fit in a single wave.
  // CTAs per item: 128-row groups on the tcgen05 kernel, 256-row groups on the dual one
  // (per video, as the CTA list gives each item only the groups its video's rows need;
  // the fused tail keeps one dense grid of the largest count)
  const int rows_per_cta = (kern == PAD_FLAG_PREFIX_TC) ? 128 : (kern == PAD_FLAG_PREFIX_DUAL) ? 256 : 0;
  const int groups = rows_per_cta ? std::max(1, (max_rows + rows_per_cta - 1) / rows_per_cta) : 1;
  const bool want_fused = kern == PAD_FLAG_PREFIX_TC && (prob->flags & PAD_FLAG_FUSED_MERGE);
  auto groups_of = [&](int b) {
    if (!rows_per_cta || want_fused) return groups;
    return std::max(1, (L->ev_count[b] * L->group + rows_per_cta - 1) / rows_per_cta);
  };
  int64_t work = 0;
  for (int b = 0; b < n_videos; ++b)
    if (L->ev_count[b] > 0) work += (int64_t)prefix_len[b] * prob->h_kv * groups_of(b);
  const int64_t target = std::max(1, n_sms);
  int64_t chunk = (work + target - 1) / target;
  chunk = std::max<int64_t>(kSplitGranule, (chunk + kSplitGranule - 1) / kSplitGranule * kSplitGranule);
  auto ctas_for = [&](int64_t c) {
    int64_t n = 0;
    for (int b = 0; b < n_videos; ++b)
      if (L->ev_count[b] > 0 && prefix_len[b] > 0)
        n += (int64_t)prob->h_kv * ((prefix_len[b] + c - 1) / c) * groups_of(b);
    return n;
  };
  if (kern == PAD_FLAG_PREFIX_TC || kern == PAD_FLAG_PREFIX_DUAL) {
    int64_t max_prefix = 0;
    for (int b = 0; b < n_videos; ++b)
      if (L->ev_count[b] > 0) max_prefix = std::max<int64_t>(max_prefix, prefix_len[b]);
    while (ctas_for(chunk) > target && chunk < max_prefix) chunk += kSplitGranule;
    // The branch/merge CTAs (one per event and kv-head) do their part before the grid wait
    // (staging, the append and, in a one-call step, the whole branch pass) during the prefix
    // pass only on SMs the prefix grid leaves free; the others do it after the prefix CTAs
    // retire.  A split up to two tiles longer is taken when it leaves room for every task and
    // its extra tiles cost less than that serial part.  Costs measured on GB300: ~0.85 us per
    // 128-token tile of a CTA in steady state, ~2 us for a task's part before the wait.
    if (!want_fused) {
      constexpr double kTileUs = 0.85, kTaskPreWaitUs = 2.0;
      const int64_t tasks = (int64_t)n_events * prob->h_kv;
      auto cost = [&](int64_t c) {
        const int64_t n_free = target - ctas_for(c);
        return (double)((c + kSplitGranule - 1) / kSplitGranule) * kTileUs + (tasks > n_free ? kTaskPreWaitUs : 0.0);
      };
      int64_t best = chunk;
      double best_cost = cost(chunk);
      for (int64_t c = chunk + kSplitGranule; c <= std::min<int64_t>(max_prefix, chunk + 2 * kSplitGranule);
           c += kSplitGranule) {
        const double v = cost(c);
        if (v < best_cost) {
          best = c;
          best_cost = v;
        }
      }
      chunk = best;
    }
  }
  if (chunk > (int64_t)1 << 30) return fail(PAD_ERR_UNSUPPORTED, "prefix too long");
  // Per-video splits for a batch of videos on the tensor-core kernels.  One split length for
  // all, sized to one wave, gives the longest video's CTAs the most tiles while a short
  // video's single CTA idles, and one wave leaves the splits coarse.  So the planner sizes
  // each video's splits for a grid of 1, 2 or 3 waves: every video starts with one split per
  // (kv-head, row group), and the video whose CTAs hold the most tiles takes one more split
  // while the grid has room.  Each candidate is costed by list-scheduling its CTAs, longest
  // first, onto the SMs (a CTA costs kCtaUs of set-up and drain plus kTileUs per tile,
  // measured on GB300), and the cheapest is kept; the CTA list is then ordered longest first.
  // The decision depends only on the batch's shape, so the last one is reused.
  L->vsplit.assign(n_videos, chunk);
  L->longest_first = false;
  if ((kern == PAD_FLAG_PREFIX_TC || kern == PAD_FLAG_PREFIX_DUAL) && !want_fused && n_videos > 1) {
    constexpr double kTileUs = 0.85, kCtaUs = 4.0;
    std::vector<int64_t> tiles(n_videos, 0), units(n_videos, 0);
    int64_t base_ctas = 0;
    for (int b = 0; b < n_videos; ++b) {
      if (L->ev_count[b] == 0 || prefix_len[b] == 0) continue;
      tiles[b] = (prefix_len[b] + kSplitGranule - 1) / kSplitGranule;
      units[b] = (int64_t)prob->h_kv * groups_of(b);
      base_ctas += units[b];
    }
    thread_local std::vector<int64_t> memo_key, memo_split;
    std::vector<int64_t> key;
    key.reserve(2 * (size_t)n_videos + 3);
    key.push_back(target);
    key.push_back(chunk);
    key.push_back(prob->flags);
    for (int b = 0; b < n_videos; ++b) {
      key.push_back(tiles[b]);
      key.push_back(units[b]);
    }
    if (key == memo_key) {
      L->vsplit = memo_split;
    } else if (base_ctas <= 3 * target) {
      auto split_for = [&](int64_t budget, std::vector<int64_t>& ns) {
        ns.assign(n_videos, 0);
        std::priority_queue<std::pair<int64_t, int>> pq;  // (tiles per CTA, video)
        for (int b = 0; b < n_videos; ++b)
          if (tiles[b] > 0) {
            ns[b] = 1;
            pq.push({tiles[b], b});
          }
        budget -= base_ctas;
        while (!pq.empty()) {
          const int top = pq.top().second;
          if (tiles[top] <= ns[top] || units[top] > budget) break;
          pq.pop();
          ++ns[top];
          budget -= units[top];
          pq.push({(tiles[top] + ns[top] - 1) / ns[top], top});
        }
      };
      auto makespan = [&](const std::vector<int64_t>& ns) {
        std::vector<std::pair<int64_t, int64_t>> durs;  // (tiles, CTA count), longest first
        for (int b = 0; b < n_videos; ++b) {
          if (ns[b] == 0) continue;
          const int64_t per = (tiles[b] + ns[b] - 1) / ns[b], n = (tiles[b] + per - 1) / per;
          durs.push_back({per, units[b] * (n - 1)});
          durs.push_back({tiles[b] - per * (n - 1), units[b]});
        }
        std::sort(durs.begin(), durs.end(),
                  [](const std::pair<int64_t, int64_t>& x, const std::pair<int64_t, int64_t>& y) {
                    return x.first > y.first;
                  });
        std::priority_queue<double, std::vector<double>, std::greater<double>> sm;
        for (int64_t i = 0; i < target; ++i) sm.push(0.0);
        double end = 0.0;
        for (const auto& d : durs)
          for (int64_t k = 0; k < d.second; ++k) {
            const double t = sm.top() + kCtaUs + kTileUs * (double)d.first;
            sm.pop();
            sm.push(t);
            end = std::max(end, t);
          }
        return end;
      };
      // the one-split-length plan as the baseline
      std::vector<int64_t> ns_global(n_videos, 0);
      const int64_t chunk_tiles = chunk / kSplitGranule;
      for (int b = 0; b < n_videos; ++b)
        if (tiles[b] > 0) ns_global[b] = (tiles[b] + chunk_tiles - 1) / chunk_tiles;
      double best = makespan(ns_global);
      std::vector<int64_t> ns, best_ns;
      for (int waves = 1; waves <= 3; ++waves) {
        if (base_ctas > waves * target) continue;
        split_for(waves * target, ns);
        const double v = makespan(ns);
        if (v < best) {
          best = v;
          best_ns = ns;
        }
      }
      if (!best_ns.empty())
        for (int b = 0; b < n_videos; ++b)
          if (best_ns[b] > 0) L->vsplit[b] = (tiles[b] + best_ns[b] - 1) / best_ns[b] * kSplitGranule;
      memo_key = key;
      memo_split = L->vsplit;
    }
    L->longest_first = true;
  }
  int64_t longest = 0;
  for (int b = 0; b < n_videos; ++b)
    if (L->ev_count[b] > 0 && prefix_len[b] > 0) longest = std::max(longest, L->vsplit[b]);
  L->split_len = (int)(longest > 0 ? longest : chunk);
  int64_t items = 0, rows = 0;
  for (int b = 0; b < n_videos; ++b) {
    if (L->ev_count[b] == 0 || prefix_len[b] == 0) continue;
    const int64_t vs = L->vsplit[b];
    const int ns = (int)((prefix_len[b] + vs - 1) / vs);
    if (ns > 32767) return fail(PAD_ERR_UNSUPPORTED, "too many splits for video %d", b);
    L->n_splits[b] = ns;
    if (rows > INT32_MAX) return fail(PAD_ERR_UNSUPPORTED, "partial rows exceed int32");
    L->part_base[b] = (int32_t)rows;
    items += (int64_t)ns * prob->h_kv;
    rows += (int64_t)prob->h_kv * ns * L->ev_count[b] * L->group;
  }
  if (rows > INT32_MAX || items > INT32_MAX) return fail(PAD_ERR_UNSUPPORTED, "batch too large");
  L->n_items = items;
  L->partial_rows = rows;

  // Fused tail: when every (event, kv-head) task can go to a prefix CTA of its own, the
  // tensor-core kernel runs a4 + a5 after its split (tasks go first to the CTAs with the
  // shortest splits, which finish first) and no separate merge kernel is launched.
  L->cnt_base.assign(n_videos, 0);
  L->n_counters = 0;
  L->fused = false;
  L->n_ctas = 0;
  L->cta_task.clear();
  if (kern == PAD_FLAG_PREFIX_TC && items > 0 && (prob->flags & PAD_FLAG_FUSED_MERGE) &&
      items * groups <= (int64_t)std::max(1, n_sms)) {
    // (the tail waits for other CTAs' splits: the whole grid must be resident at once,
    // which one CTA per SM and a grid of at most one wave guarantee)
    L->n_ctas = items * groups;
    std::vector<std::pair<int64_t, int64_t>> valid;  // (split tokens, CTA index)
    int64_t item = 0;
    for (int b = 0; b < n_videos; ++b) {
      if (L->ev_count[b] == 0 || L->n_splits[b] == 0) continue;
      const int R = L->ev_count[b] * L->group;
      const int gb = (R + 127) / 128;
      L->cnt_base[b] = (int32_t)L->n_counters;
      L->n_counters += (int64_t)prob->h_kv * gb;
      for (int h = 0; h < prob->h_kv; ++h)
        for (int s = 0; s < L->n_splits[b]; ++s, ++item) {
          const int64_t tok = std::min<int64_t>(prefix_len[b], (int64_t)(s + 1) * chunk) - (int64_t)s * chunk;
          for (int g = 0; g < gb; ++g) valid.push_back({tok, item * groups + g});
        }
    }
    const int64_t tasks_n = (int64_t)n_events * prob->h_kv;
    if (tasks_n <= (int64_t)valid.size()) {
      std::stable_sort(valid.begin(), valid.end(),
                       [](const std::pair<int64_t, int64_t>& x, const std::pair<int64_t, int64_t>& y) {
                         return x.first < y.first;
                       });
      L->cta_task.assign(L->n_ctas, -1);
      for (int64_t t = 0; t < tasks_n; ++t) L->cta_task[valid[t].second] = (int32_t)t;
      L->fused = true;
    }
  }
  L->cta_map = false;
  if (rows_per_cta && !L->fused && items > 0) {
    if (items > ((int64_t)1 << 24)) return fail(PAD_ERR_UNSUPPORTED, "batch too large");
    L->cta_task.clear();
    std::vector<std::pair<int64_t, int32_t>> order;  // (split tokens, CTA entry)
    int64_t item = 0;
    for (int b = 0; b < n_videos; ++b) {
      if (L->ev_count[b] == 0 || L->n_splits[b] == 0) continue;
      const int gb = groups_of(b);
      const int64_t vs = L->vsplit[b];
      for (int h = 0; h < prob->h_kv; ++h)
        for (int sp = 0; sp < L->n_splits[b]; ++sp, ++item) {
          const int64_t tok = std::min<int64_t>(prefix_len[b], (sp + 1) * vs) - sp * vs;
          for (int g = 0; g < gb; ++g) order.push_back({tok, (int32_t)((item << 6) | g)});
        }
    }
    // a batch of videos: the longest splits start first
    if (L->longest_first)
      std::stable_sort(order.begin(), order.end(),
                       [](const std::pair<int64_t, int32_t>& x, const std::pair<int64_t, int32_t>& y) {
                         return x.first > y.first;
                       });
    L->cta_task.reserve(order.size());
    for (const auto& o : order) L->cta_task.push_back(o.second);
    L->n_ctas = (int64_t)L->cta_task.size();
    L->cta_map = true;
  }
  // A branch/merge CTA that starts beside the prefix grid runs its branch pass there, then
  // holds its slot until that grid completes; with a one-wave tensor-core grid, the slots
  // beside it are those of the SMs it leaves free (two CTAs each).  When some (event,
  // kv-head) task gets none, it starts only once the prefix CTAs leave, and the whole step
  // then waits for its branch pass and merge in series: there every task waits for the
  // prefix grid first and stages the split partials while its branch pass runs.
  L->merge_first = false;
  if (kern == PAD_FLAG_PREFIX_TC && !L->fused && L->n_ctas > 0 && L->n_ctas <= n_sms) {
    const int64_t free_slots = 2 * ((int64_t)n_sms - L->n_ctas);
    L->merge_first = (int64_t)n_events * prob->h_kv > free_slots;
  }

  size_t off = sizeof(PadDevHeader);
  L->off_videos = off;
  off = align_up(off + (size_t)n_videos * sizeof(PadVideoDesc), 256);
  L->off_events = off;
  off = align_up(off + (size_t)n_events * sizeof(PadEventDesc), 256);
  L->off_items = off;
  off = off + (size_t)items * sizeof(PadWorkItem);
  L->off_tasks = off;
  off = off + (size_t)L->cta_task.size() * sizeof(int32_t);
  L->upload_bytes = off;
  off = align_up(off, 256);
  L->off_ml = off;
  off = align_up(off + (size_t)rows * sizeof(float2), 256);
  L->off_o = off;
  off = align_up(off + (size_t)rows * prob->head_dim * sizeof(float), 256);
  L->off_cnt = off;
  off = align_up(off + (size_t)L->n_counters * sizeof(unsigned int), 256);
  L->total_bytes = off;
  return PAD_OK;
}

// Plan images in pinned, device-mapped host memory.  The kernels read a plan's video and
// event descriptors and its work items in place, so a step puts no copy on the stream
// between the previous step's last kernel and its own first one.  An image belongs to
// its plan until pad_plan_destroy; it then joins its device's FIFO and is rewritten only
// after the event recorded behind the last launch that read it has completed.  Up to
// kImagesInFlight images per device are cycled; more are allocated while plans are held.
struct PlanImage {
  void* host = nullptr;
  void* dev = nullptr;
  size_t cap = 0;
  cudaEvent_t done = nullptr;
  bool recorded = false;
  int device = 0;
};
constexpr int kImagesInFlight = 8;
struct ImagePool {
  std::mutex mu;
  std::deque<PlanImage*> fifo;
  int count = 0;
};
ImagePool g_images[64];

cudaError_t image_alloc(PlanImage* img, size_t n) {
  if (img->host) cudaFreeHost(img->host);
  img->host = img->dev = nullptr;
  img->cap = 0;
  const size_t cap = std::max<size_t>(n, 64 * 1024);
  cudaError_t e = cudaHostAlloc(&img->host, cap, cudaHostAllocMapped | cudaHostAllocPortable);
  if (e != cudaSuccess) return e;
  e = cudaHostGetDevicePointer(&img->dev, img->host, 0);
  if (e != cudaSuccess) return e;
  img->cap = cap;
  return cudaSuccess;
}

cudaError_t image_acquire(size_t n, PlanImage** out) {
  *out = nullptr;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  ImagePool& pool = g_images[dev];
  PlanImage* img = nullptr;
  {
    std::lock_guard<std::mutex> lk(pool.mu);
    if (pool.count >= kImagesInFlight && !pool.fifo.empty()) {
      img = pool.fifo.front();
      pool.fifo.pop_front();
    } else {
      ++pool.count;
    }
  }
  if (!img) {
    img = new PlanImage();
    img->device = dev;
    e = cudaEventCreateWithFlags(&img->done, cudaEventDisableTiming);
    if (e == cudaSuccess) e = image_alloc(img, n);
  } else {
    if (img->recorded) e = cudaEventSynchronize(img->done);
    img->recorded = false;
    if (e == cudaSuccess && img->cap < n) e = image_alloc(img, n);
  }
  if (e != cudaSuccess) {
    std::lock_guard<std::mutex> lk(pool.mu);
    pool.fifo.push_back(img);
    return e;
  }
  *out = img;
  return cudaSuccess;
}

void image_release(PlanImage* img) {
  if (!img) return;
  ImagePool& pool = g_images[img->device];
  std::lock_guard<std::mutex> lk(pool.mu);
  pool.fifo.push_back(img);
}

// Generations of plans: 56-bit, nonzero, from a per-process random start.
uint64_t next_generation() {
  static std::atomic<uint64_t> ctr{0};
  static const uint64_t base = [] {
    std::random_device rd;
    return ((uint64_t)rd() << 32) ^ (uint64_t)rd() ^
           (uint64_t)std::chrono::steady_clock::now().time_since_epoch().count();
  }();
  for (;;) {
    const uint64_t g = (base + ctr.fetch_add(1)) & ((1ull << 56) - 1);
    if (g != 0) return g;
  }
}

// Timing of the dominant kernel (process-global measurement aid).
struct Timing {
  bool on = false;
  int max = 0;
  int n = 0;
  std::vector<cudaEvent_t> ev;
};
Timing g_timing;

}  // namespace

// ---------------------------------------------------------------------------
// Page pool bookkeeping
// ---------------------------------------------------------------------------
struct pad_cache_state {
  int32_t n_pages = 0;
  int32_t free_count = 0;
  std::vector<uint64_t> used;  // bit p set = page p in use

  bool is_used(int p) const { return (used[p >> 6] >> (p & 63)) & 1u; }
  void set(int p, bool u) {
    if (u)
      used[p >> 6] |= (uint64_t)1 << (p & 63);
    else
      used[p >> 6] &= ~((uint64_t)1 << (p & 63));
  }
  // Lowest-numbered free page >= from, or -1.
  int next_free(int from) const {
    if (from >= n_pages) return -1;
    size_t w = (size_t)from >> 6;
    uint64_t bits = ~used[w] & (~(uint64_t)0 << (from & 63));
    while (true) {
      if (bits) {
        int p = (int)(w * 64 + __builtin_ctzll(bits));
        return p < n_pages ? p : -1;
      }
      if (++w >= used.size()) return -1;
      bits = ~used[w];
    }
  }
};

struct pad_plan_t {
  pad_problem prob{};
  Layout lay;
  int32_t n_videos = 0, n_events = 0;
  int32_t max_pages = 0, n_pages = 0;
  int32_t max_event_len = 0;        // longest branch (private tokens before this step)
  int32_t* page_table = nullptr;
  void* workspace = nullptr;
  int64_t total_prefix_tokens = 0;
  int32_t n_new_pages = 0;
  std::vector<int32_t> new_pages;
  std::vector<uint8_t> host_image;  // header + videos + events + items
  PlanImage* image = nullptr;       // the same bytes in pinned memory, read by the kernels
                                    // when they do not fit the launch parameters
  std::vector<uint8_t> param_image; // videos | events | items, packed, for KParams::img
  int32_t img_videos = 0, img_events = 0, img_items = 0, img_tasks = 0;
  const float* rope_cs = nullptr;   // rotary table (pad_plan_set_rope), else NULL
  int32_t g_self = 0;               // self G-token mask (pad_plan_set_g_visibility)
  int32_t causal = 0;               // causal mask (pad_plan_set_branch_visibility)
  int32_t task_keys = 0;            // most keys one branch task reads (set with causal)
  uint64_t gen = 0;                 // generation tagging this plan's device errors
  ~pad_plan_t() { image_release(image); }
};

extern "C" {

const char* pad_last_error(void) { return g_last_error.c_str(); }

const char* pad_status_string(pad_status s) {
  switch (s) {
    case PAD_OK: return "PAD_OK";
    case PAD_ERR_INVALID_ARG: return "PAD_ERR_INVALID_ARG";
    case PAD_ERR_UNSUPPORTED: return "PAD_ERR_UNSUPPORTED";
    case PAD_ERR_OUT_OF_PAGES: return "PAD_ERR_OUT_OF_PAGES";
    case PAD_ERR_WORKSPACE_TOO_SMALL: return "PAD_ERR_WORKSPACE_TOO_SMALL";
    case PAD_ERR_CUDA: return "PAD_ERR_CUDA";
    case PAD_ERR_DEVICE_TIMEOUT: return "PAD_ERR_DEVICE_TIMEOUT";
    case PAD_ERR_DEVICE_BOUNDS: return "PAD_ERR_DEVICE_BOUNDS";
  }
  return "PAD_ERR_UNKNOWN";
}

pad_status pad_cache_state_create(int32_t n_pages, pad_cache_state** out) {
  if (!out) return fail(PAD_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  if (n_pages < 0) return fail(PAD_ERR_INVALID_ARG, "n_pages=%d < 0", n_pages);
  auto* c = new pad_cache_state();
  c->n_pages = n_pages;
  c->free_count = n_pages;
  c->used.assign(((size_t)n_pages + 63) / 64 + 1, 0);
  *out = c;
  return PAD_OK;
}

void pad_cache_state_destroy(pad_cache_state* cache) { delete cache; }

int32_t pad_cache_state_num_pages(const pad_cache_state* c) { return c ? c->n_pages : -1; }
int32_t pad_cache_state_free_count(const pad_cache_state* c) { return c ? c->free_count : -1; }

static pad_status set_pages(pad_cache_state* c, const int32_t* pages, int32_t n, bool to_used) {
  if (!c) return fail(PAD_ERR_INVALID_ARG, "cache is NULL");
  if (n < 0 || (n > 0 && !pages)) return fail(PAD_ERR_INVALID_ARG, "bad page list");
  std::vector<int32_t> seen(pages, pages + n);
  std::sort(seen.begin(), seen.end());
  for (int i = 0; i < n; ++i) {
    const int p = seen[i];
    if (p < 0 || p >= c->n_pages) return fail(PAD_ERR_INVALID_ARG, "page %d outside [0, %d)", p, c->n_pages);
    if (i > 0 && seen[i - 1] == p) return fail(PAD_ERR_INVALID_ARG, "page %d listed twice", p);
    if (c->is_used(p) == to_used)
      return fail(PAD_ERR_INVALID_ARG, "page %d is already %s", p, to_used ? "in use" : "free");
  }
  for (int i = 0; i < n; ++i) c->set(pages[i], to_used);
  c->free_count += to_used ? -n : n;
  return PAD_OK;
}

pad_status pad_cache_state_mark_used(pad_cache_state* c, const int32_t* pages, int32_t n) {
  return set_pages(c, pages, n, true);
}

pad_status pad_cache_state_release(pad_cache_state* c, const int32_t* pages, int32_t n) {
  return set_pages(c, pages, n, false);
}

pad_status pad_cache_state_export(const pad_cache_state* c, uint8_t* used) {
  if (!c || (!used && c->n_pages > 0)) return fail(PAD_ERR_INVALID_ARG, "NULL argument");
  for (int p = 0; p < c->n_pages; ++p) used[p] = c->is_used(p) ? 1 : 0;
  return PAD_OK;
}

pad_status pad_cache_state_import(pad_cache_state* c, const uint8_t* used, int32_t n_pages) {
  if (!c || (!used && n_pages > 0)) return fail(PAD_ERR_INVALID_ARG, "NULL argument");
  if (n_pages != c->n_pages)
    return fail(PAD_ERR_INVALID_ARG, "checkpoint has %d pages, pool has %d", n_pages, c->n_pages);
  int fc = 0;
  for (int p = 0; p < n_pages; ++p) {
    if (used[p] > 1) return fail(PAD_ERR_INVALID_ARG, "used[%d]=%d is not 0/1", p, used[p]);
  }
  for (int p = 0; p < n_pages; ++p) {
    c->set(p, used[p] != 0);
    fc += used[p] == 0;
  }
  c->free_count = fc;
  return PAD_OK;
}

size_t pad_workspace_size(const pad_problem* prob, int32_t n_videos, const int32_t* prefix_len,
                          int32_t n_events, const int32_t* event_video) {
  if (check_problem(prob) != PAD_OK) return 0;
  Layout L;
  const int sms = prob->num_sms > 0 ? prob->num_sms : query_num_sms();
  if (compute_layout(prob, n_videos, prefix_len, n_events, event_video, sms, &L) != PAD_OK) return 0;
  return L.total_bytes;
}

pad_status pad_plan(const pad_problem* prob, pad_cache_state* cache, int32_t n_videos,
                    const int32_t* prefix_len, const int64_t* prefix_offset, int32_t n_events,
                    const int32_t* event_video, const int32_t* event_len, int32_t* page_table,
                    int32_t max_pages, void* workspace, size_t workspace_bytes,
                    pad_stream_t stream, pad_plan_t** plan_out) {
  NvtxRange nvtx_range("pad_plan");
  if (!plan_out) return fail(PAD_ERR_INVALID_ARG, "plan_out is NULL");
  *plan_out = nullptr;
  pad_status st = check_problem(prob);
  if (st != PAD_OK) return st;
  if (!cache) return fail(PAD_ERR_INVALID_ARG, "cache is NULL");
  if (n_events > 0 && !event_len) return fail(PAD_ERR_INVALID_ARG, "event_len is NULL");
  if (max_pages <= 0 && n_events > 0) return fail(PAD_ERR_INVALID_ARG, "max_pages must be > 0");
  if (workspace && (reinterpret_cast<uintptr_t>(workspace) & 255u))
    return fail(PAD_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
  if (workspace && n_events > 0 && !page_table)
    return fail(PAD_ERR_INVALID_ARG, "page_table is NULL");

  const int sms = prob->num_sms > 0 ? prob->num_sms : (workspace ? query_num_sms() : kDefaultSms);
  auto* plan = new pad_plan_t();
  Layout& L = plan->lay;
  st = compute_layout(prob, n_videos, prefix_len, n_events, event_video, sms, &L);
  if (st != PAD_OK) {
    delete plan;
    return st;
  }
  if (workspace && workspace_bytes < L.total_bytes) {
    delete plan;
    return fail(PAD_ERR_WORKSPACE_TOO_SMALL, "workspace has %zu bytes, plan needs %zu",
                workspace_bytes, L.total_bytes);
  }
  const int ps = prob->page_size;
  int need = 0;
  for (int e = 0; e < n_events; ++e) {
    const int len = event_len[e];
    if (len < 0) {
      delete plan;
      return fail(PAD_ERR_INVALID_ARG, "event_len[%d]=%d < 0", e, len);
    }
    if (len > 65534) {
      delete plan;
      return fail(PAD_ERR_UNSUPPORTED, "event_len[%d]=%d: branches hold at most 65535 tokens", e, len);
    }
    if (len / ps >= max_pages) {
      delete plan;
      return fail(PAD_ERR_INVALID_ARG, "event %d: length %d needs page index %d >= max_pages=%d", e,
                  len, len / ps, max_pages);
    }
    need += (len % ps) == 0;
  }
  if (need > cache->free_count) {
    delete plan;
    return fail(PAD_ERR_OUT_OF_PAGES, "step needs %d new pages, %d free", need, cache->free_count);
  }

  // Host image of the device plan.
  std::vector<PadVideoDesc> vids(n_videos);
  int64_t packed = 0, total_tokens = 0;
  for (int b = 0; b < n_videos; ++b) {
    int64_t off = prefix_offset ? prefix_offset[b] : packed;
    if (off < 0) {
      delete plan;
      return fail(PAD_ERR_INVALID_ARG, "prefix_offset[%d] < 0", b);
    }
    packed += prefix_len[b];
    total_tokens = std::max(total_tokens, off + prefix_len[b]);
    PadVideoDesc& v = vids[b];
    v.prefix_off = off;
    v.prefix_len = prefix_len[b];
    v.first_event = L.ev_first[b];
    v.n_events = L.ev_count[b];
    v.n_splits = (int16_t)L.n_splits[b];
    v.n_planning = 0;
    v.part_base = L.part_base[b];
    v.cnt_base = L.cnt_base[b];
  }
  std::vector<PadWorkItem> items;
  items.reserve(L.n_items);
  for (int b = 0; b < n_videos; ++b) {
    for (int h = 0; h < prob->h_kv; ++h) {
      for (int s = 0; s < L.n_splits[b]; ++s) {
        PadWorkItem it;
        const int32_t vs = (int32_t)L.vsplit[b];
        it.tok_begin = s * vs;
        it.tok_end = std::min(prefix_len[b], (s + 1) * vs);
        it.tok0 = vids[b].prefix_off + it.tok_begin;
        it.first_event = L.ev_first[b];
        it.n_events = L.ev_count[b];
        it.part_row0 = L.part_base[b] + (h * L.n_splits[b] + s) * (L.ev_count[b] * L.group);
        it.kvh = (int16_t)h;
        it.split = (int16_t)s;
        items.push_back(it);
      }
    }
  }

  // Page allocation: ascending events, lowest free page first.
  std::vector<PadEventDesc> evs(n_events);
  plan->new_pages.assign(n_events, -1);
  int cursor = 0;
  for (int e = 0; e < n_events; ++e) {
    PadEventDesc& d = evs[e];
    d.video = (uint16_t)event_video[e];
    d.len = (uint16_t)event_len[e];
    d.local = (uint16_t)(e - L.ev_first[event_video[e]]);
    d.new_page = -1;
    d.pos = 0;
    d.gidx = 0;
    if (event_len[e] % ps == 0) {
      const int pg = cache->next_free(cursor);
      // need <= free_count guarantees a page exists
      d.new_page = pg;
      plan->new_pages[e] = pg;
      cache->set(pg, true);
      cursor = pg + 1;
    }
  }
  cache->free_count -= need;

  PadDevHeader hdr;
  std::memset(&hdr, 0, sizeof(hdr));
  plan->host_image.assign(L.upload_bytes, 0);
  std::memcpy(plan->host_image.data(), &hdr, sizeof(hdr));
  if (n_videos) std::memcpy(plan->host_image.data() + L.off_videos, vids.data(), vids.size() * sizeof(PadVideoDesc));
  if (n_events) std::memcpy(plan->host_image.data() + L.off_events, evs.data(), evs.size() * sizeof(PadEventDesc));
  if (!items.empty())
    std::memcpy(plan->host_image.data() + L.off_items, items.data(), items.size() * sizeof(PadWorkItem));
  if (!L.cta_task.empty())
    std::memcpy(plan->host_image.data() + L.off_tasks, L.cta_task.data(), L.cta_task.size() * sizeof(int32_t));

  plan->gen = next_generation();
  {
    const size_t nv = vids.size() * sizeof(PadVideoDesc), ne = evs.size() * sizeof(PadEventDesc);
    const size_t ni = items.size() * sizeof(PadWorkItem);
    const size_t nt = L.cta_task.size() * sizeof(int32_t);
    plan->img_videos = 0;
    plan->img_events = (int32_t)align_up(nv, 16);
    plan->img_items = (int32_t)(plan->img_events + align_up(ne, 16));
    plan->img_tasks = (int32_t)(plan->img_items + align_up(ni, 16));
    const size_t total = plan->img_tasks + nt;
    if (n_events > 0 && total <= (size_t)kParamImageBytes) {
      plan->param_image.assign(total, 0);
      if (nv) std::memcpy(plan->param_image.data(), vids.data(), nv);
      if (ne) std::memcpy(plan->param_image.data() + plan->img_events, evs.data(), ne);
      if (ni) std::memcpy(plan->param_image.data() + plan->img_items, items.data(), ni);
      if (nt) std::memcpy(plan->param_image.data() + plan->img_tasks, L.cta_task.data(), nt);
    }
  }
  if (workspace && n_events > 0 && plan->param_image.empty()) {
    cudaError_t ce = image_acquire(L.upload_bytes, &plan->image);
    if (ce != cudaSuccess) {
      for (int e = 0; e < n_events; ++e)
        if (plan->new_pages[e] >= 0) cache->set(plan->new_pages[e], false);
      cache->free_count += need;
      delete plan;
      return cuda_fail(ce, "plan image");
    }
    std::memcpy(plan->image->host, plan->host_image.data(), L.upload_bytes);
  }
  plan->prob = *prob;
  plan->n_videos = n_videos;
  plan->n_events = n_events;
  plan->max_event_len = 0;
  for (int e = 0; e < n_events; ++e) plan->max_event_len = std::max(plan->max_event_len, event_len[e]);
  plan->max_pages = max_pages;
  plan->n_pages = cache->n_pages;
  plan->page_table = page_table;
  plan->workspace = workspace;
  plan->total_prefix_tokens = total_tokens;
  plan->n_new_pages = need;
  *plan_out = plan;
  return PAD_OK;
}

pad_status pad_plan_set_rope(pad_plan_t* plan, const int32_t* positions, const float* cos_sin,
                             int32_t max_position) {
  if (!plan) return fail(PAD_ERR_INVALID_ARG, "plan is NULL");
  if (!cos_sin) return fail(PAD_ERR_INVALID_ARG, "cos_sin is NULL");
  if (!aligned16(cos_sin)) return fail(PAD_ERR_INVALID_ARG, "cos_sin must be 16-byte aligned");
  if (max_position <= 0) return fail(PAD_ERR_INVALID_ARG, "max_position must be > 0");
  if (plan->n_events > 0 && !positions) return fail(PAD_ERR_INVALID_ARG, "positions is NULL");
  for (int e = 0; e < plan->n_events; ++e)
    if (positions[e] < 0 || positions[e] >= max_position)
      return fail(PAD_ERR_INVALID_ARG, "positions[%d]=%d outside [0, %d)", e, positions[e], max_position);
  // every copy of the event descriptors: the host image, the launch-parameter image and
  // the page-locked image (no launch of this plan has read them yet)
  auto set = [&](uint8_t* base) {
    auto* ev = reinterpret_cast<PadEventDesc*>(base);
    for (int e = 0; e < plan->n_events; ++e) ev[e].pos = positions[e];
  };
  if (plan->n_events > 0) {
    set(plan->host_image.data() + plan->lay.off_events);
    if (!plan->param_image.empty()) set(plan->param_image.data() + plan->img_events);
    if (plan->image) set(static_cast<uint8_t*>(plan->image->host) + plan->lay.off_events);
  }
  plan->rope_cs = cos_sin;
  return PAD_OK;
}

pad_status pad_plan_set_g_visibility(pad_plan_t* plan, int32_t mode, const int32_t* n_planning,
                                     const int32_t* g_index) {
  if (!plan) return fail(PAD_ERR_INVALID_ARG, "plan is NULL");
  if (mode != PAD_G_ALL && mode != PAD_G_SELF) return fail(PAD_ERR_INVALID_ARG, "mode %d", mode);
  std::vector<int32_t> K(plan->n_videos, 0), gi(plan->n_events, 0);
  if (mode == PAD_G_SELF) {
    if ((plan->n_videos > 0 && !n_planning) || (plan->n_events > 0 && !g_index))
      return fail(PAD_ERR_INVALID_ARG, "n_planning / g_index is NULL");
    auto* vids = reinterpret_cast<const PadVideoDesc*>(plan->host_image.data() + plan->lay.off_videos);
    auto* evs = reinterpret_cast<const PadEventDesc*>(plan->host_image.data() + plan->lay.off_events);
    for (int b = 0; b < plan->n_videos; ++b) {
      if (n_planning[b] < 0 || n_planning[b] > 32767 || n_planning[b] + 1 > std::max(1, vids[b].prefix_len))
        return fail(PAD_ERR_INVALID_ARG, "n_planning[%d]=%d: the prefix (%d tokens) must hold G^1..G^K and S", b,
                    n_planning[b], vids[b].prefix_len);
      K[b] = n_planning[b];
    }
    for (int e = 0; e < plan->n_events; ++e) {
      const int v = evs[e].video;
      if (g_index[e] < 0 || g_index[e] >= std::max(1, K[v]) || (K[v] == 0 && g_index[e] != 0))
        return fail(PAD_ERR_INVALID_ARG, "g_index[%d]=%d outside [0, %d)", e, g_index[e], K[v]);
      gi[e] = g_index[e];
    }
  }
  // every copy of the descriptors (no launch of this plan has read them yet)
  auto set = [&](uint8_t* vbase, uint8_t* ebase) {
    auto* v = reinterpret_cast<PadVideoDesc*>(vbase);
    auto* ev = reinterpret_cast<PadEventDesc*>(ebase);
    for (int b = 0; b < plan->n_videos; ++b) v[b].n_planning = (int16_t)K[b];
    for (int e = 0; e < plan->n_events; ++e) ev[e].gidx = (uint16_t)gi[e];
  };
  if (plan->n_events > 0) {
    set(plan->host_image.data() + plan->lay.off_videos, plan->host_image.data() + plan->lay.off_events);
    if (!plan->param_image.empty())
      set(plan->param_image.data() + plan->img_videos, plan->param_image.data() + plan->img_events);
    if (plan->image)
      set(static_cast<uint8_t*>(plan->image->host) + plan->lay.off_videos,
          static_cast<uint8_t*>(plan->image->host) + plan->lay.off_events);
  }
  plan->g_self = mode == PAD_G_SELF ? 1 : 0;
  return PAD_OK;
}

pad_status pad_plan_set_branch_visibility(pad_plan_t* plan, int32_t mode) {
  if (!plan) return fail(PAD_ERR_INVALID_ARG, "plan is NULL");
  if (mode != PAD_BRANCH_OWN && mode != PAD_BRANCH_CAUSAL) return fail(PAD_ERR_INVALID_ARG, "mode %d", mode);
  int64_t most = 0;
  if (plan->n_events > 0) {
    auto* vids = reinterpret_cast<const PadVideoDesc*>(plan->host_image.data() + plan->lay.off_videos);
    auto* evs = reinterpret_cast<const PadEventDesc*>(plan->host_image.data() + plan->lay.off_events);
    for (int b = 0; b < plan->n_videos; ++b) {
      int64_t sum = 1;
      for (int f = 0; f < vids[b].n_events; ++f) sum += evs[vids[b].first_event + f].len;
      most = std::max(most, sum);
    }
  }
  if (most > INT32_MAX) return fail(PAD_ERR_UNSUPPORTED, "too many branch tokens in one video");
  plan->causal = mode == PAD_BRANCH_CAUSAL ? 1 : 0;
  plan->task_keys = (int32_t)most;
  return PAD_OK;
}

pad_status pad_plan_new_pages(const pad_plan_t* plan, int32_t* new_page) {
  if (!plan || (!new_page && plan->n_events > 0)) return fail(PAD_ERR_INVALID_ARG, "NULL argument");
  std::copy(plan->new_pages.begin(), plan->new_pages.end(), new_page);
  return PAD_OK;
}

pad_status pad_plan_release_new_pages(const pad_plan_t* plan, pad_cache_state* cache) {
  if (!plan || !cache) return fail(PAD_ERR_INVALID_ARG, "NULL argument");
  std::vector<int32_t> pages;
  for (int32_t pg : plan->new_pages)
    if (pg >= 0) pages.push_back(pg);
  return pages.empty() ? PAD_OK : set_pages(cache, pages.data(), (int32_t)pages.size(), false);
}

pad_status pad_plan_get_info(const pad_plan_t* plan, pad_plan_info* info) {
  if (!plan || !info) return fail(PAD_ERR_INVALID_ARG, "NULL argument");
  info->n_videos = plan->n_videos;
  info->n_events = plan->n_events;
  info->n_work_items = (int32_t)plan->lay.n_items;
  info->split_len = plan->lay.split_len;
  info->prefix_kernel = plan->lay.prefix_kernel;
  info->n_new_pages = plan->n_new_pages;
  info->partial_rows = plan->lay.partial_rows;
  info->workspace_bytes = (int64_t)plan->lay.total_bytes;
  info->param_descriptor_bytes = (int32_t)plan->param_image.size();
  info->fused_tail = plan->lay.fused ? 1 : 0;
  info->generation = plan->gen;
  info->prefix_ctas = (int32_t)(plan->lay.n_ctas > 0 ? plan->lay.n_ctas : plan->lay.n_items);
  info->max_split_tiles = (plan->lay.split_len + kSplitGranule - 1) / kSplitGranule;
  info->merge_first = plan->lay.merge_first ? 1 : 0;
  return PAD_OK;
}

pad_status pad_plan_destroy(pad_plan_t* plan) {
  delete plan;
  return PAD_OK;
}

static pad_status static_kv_append(const pad_plan_t* plan, const void* k_new, const void* v_new, void* k_pool,
                                   void* v_pool, cudaStream_t s);
static pad_status static_status_header(PadDevHeader** out);

static void make_params(const pad_plan_t* plan, KParams& p) {
  const pad_problem& pr = plan->prob;
  p.h_q = pr.h_q;
  p.h_kv = pr.h_kv;
  p.group = pr.h_q / pr.h_kv;
  p.head_dim = pr.head_dim;
  p.page_size = pr.page_size;
  p.max_pages = plan->max_pages;
  p.n_pages = plan->n_pages;
  p.n_videos = plan->n_videos;
  p.n_events = plan->n_events;
  p.n_items = (int32_t)plan->lay.n_items;
  p.out_bf16 = pr.out_dtype == 1;
  p.n_sms = plan->lay.n_sms;
  p.max_splits = 0;
  for (int32_t ns : plan->lay.n_splits) p.max_splits = std::max(p.max_splits, ns);
  p.branch_rows = std::min(128, ((plan->causal ? plan->task_keys : plan->max_event_len + 1) + 15) / 16 * 16);
  p.scale_log2 = (float)((double)pr.scale * 1.4426950408889634);
  p.gen = plan->gen;
  auto* ws = static_cast<uint8_t*>(plan->workspace);
  p.header = reinterpret_cast<PadDevHeader*>(ws);
  p.img_n = (int32_t)plan->param_image.size();
  p.img_videos = plan->img_videos;
  p.img_events = plan->img_events;
  p.img_items = plan->img_items;
  p.img_tasks = plan->img_tasks;
  p.k_new = nullptr;
  p.v_new = nullptr;
  p.rope_cs = plan->rope_cs;
  p.g_self = plan->g_self;
  p.causal = plan->causal;
  p.fused = plan->lay.fused ? 1 : 0;
  p.cta_map = plan->lay.cta_map ? 1 : 0;
  p.n_ctas = (int32_t)plan->lay.n_ctas;
  p.tail_chunk = p.fused ? prefix_tc_tail_chunk(p.branch_rows, p.group, p.max_splits) : 0;
  p.merge_first = plan->lay.merge_first ? 1 : 0;
  p.counters = reinterpret_cast<unsigned int*>(ws + plan->lay.off_cnt);
  p.n_counters = p.fused ? (int32_t)plan->lay.n_counters : 0;
  if (p.img_n > 0) {
    std::memcpy(p.img, plan->param_image.data(), plan->param_image.size());
    p.videos = nullptr;
    p.events = nullptr;
    p.items = nullptr;
    p.tasks = nullptr;
  } else {
    auto* im = static_cast<const uint8_t*>(plan->image->dev);
    p.videos = reinterpret_cast<const PadVideoDesc*>(im + plan->lay.off_videos);
    p.events = reinterpret_cast<const PadEventDesc*>(im + plan->lay.off_events);
    p.items = reinterpret_cast<const PadWorkItem*>(im + plan->lay.off_items);
    p.tasks = reinterpret_cast<const int32_t*>(im + plan->lay.off_tasks);
  }
  p.part_ml = reinterpret_cast<float2*>(ws + plan->lay.off_ml);
  p.part_o = reinterpret_cast<float*>(ws + plan->lay.off_o);
  p.page_table = plan->page_table;
}

pad_status pad_kv_append(const pad_plan_t* plan, const void* k_new, const void* v_new,
                         void* k_pool, void* v_pool, pad_stream_t stream) {
  NvtxRange nvtx_range("pad_kv_append");
  if (!plan) return fail(PAD_ERR_INVALID_ARG, "plan is NULL");
  if (plan->n_events == 0) return PAD_OK;
  if (!k_new || !v_new || !k_pool || !v_pool) return fail(PAD_ERR_INVALID_ARG, "NULL tensor");
  if (!aligned16(k_new) || !aligned16(v_new) || !aligned16(k_pool) || !aligned16(v_pool))
    return fail(PAD_ERR_INVALID_ARG, "tensors must be 16-byte aligned");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  // a host-only plan (no workspace): the library's static scratch array stands in for it
  if (!plan->workspace) {
    if (!plan->page_table) return fail(PAD_ERR_INVALID_ARG, "plan has no page table");
    return static_kv_append(plan, k_new, v_new, k_pool, v_pool, s);
  }
  KParams p;
  make_params(plan, p);
  cudaError_t e = launch_append(p, k_new, v_new, k_pool, v_pool, s);
  if (e != cudaSuccess) return cuda_fail(e, "append launch");
  if (plan->image) {
    e = cudaEventRecord(plan->image->done, s);
    if (e != cudaSuccess) return cuda_fail(e, "plan image event");
    plan->image->recorded = true;
  }
  return PAD_OK;
}

// a3 (+ a4, a5 in the same kernel when the plan fuses them, else in the branch/merge
// kernel after it).  k_new == NULL: the append kernel ran just before (the prefix kernel
// overlaps it through programmatic dependent launch).  k_new set: no append kernel; each
// branch task appends its own row, and the prefix kernel is the step's first launch.
static pad_status launch_attention(const pad_plan_t* plan, const void* q, const void* k_new,
                                   const void* v_new, const void* k_prefix, const void* v_prefix,
                                   const void* k_pool, const void* v_pool, void* out, float* lse,
                                   pad_stream_t stream) {
  if (!plan) return fail(PAD_ERR_INVALID_ARG, "plan is NULL");
  if (plan->n_events == 0) return PAD_OK;
  if (!plan->workspace) return fail(PAD_ERR_INVALID_ARG, "plan was built without a workspace");
  if (!q || !k_pool || !v_pool || !out) return fail(PAD_ERR_INVALID_ARG, "NULL tensor");
  if (plan->lay.n_items > 0 && (!k_prefix || !v_prefix))
    return fail(PAD_ERR_INVALID_ARG, "k_prefix / v_prefix is NULL");
  if (!aligned16(q) || !aligned16(k_prefix) || !aligned16(v_prefix) || !aligned16(k_pool) ||
      !aligned16(v_pool) || !aligned16(out) || !aligned16(k_new) || !aligned16(v_new) ||
      (lse && (reinterpret_cast<uintptr_t>(lse) & 3u)))
    return fail(PAD_ERR_INVALID_ARG, "tensors must be 16-byte aligned (lse 4-byte)");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  KParams p;
  make_params(plan, p);
  p.k_new = k_new;
  p.v_new = v_new;
  const bool timed = g_timing.on && g_timing.n < g_timing.max;
  if (timed) cudaEventRecord(g_timing.ev[2 * g_timing.n], s);
  cudaError_t e = cudaSuccess;
  switch (plan->lay.prefix_kernel) {
    case PAD_FLAG_PREFIX_SIMT: e = launch_prefix_simt(p, plan->lay.max_rows, q, k_prefix, v_prefix, s); break;
    case PAD_FLAG_PREFIX_MMA: e = launch_prefix_mma(p, plan->lay.max_rows, q, k_prefix, v_prefix, s); break;
    case PAD_FLAG_PREFIX_TC:
      // programmatic dependent launch: the prefix pass overlaps the append kernel and the
      // branch/merge pass's prologue overlaps the prefix pass (not while timing events
      // are recorded between the kernels).  As the first kernel of a one-call step it
      // overlaps only the launch with the grid before it, and waits for that grid before
      // it reads or writes anything.
      e = launch_prefix_tc(p, plan->lay.max_rows, q, k_prefix, v_prefix, plan->total_prefix_tokens, k_pool,
                           v_pool, out, lse, !timed, s);
      break;
    case PAD_FLAG_PREFIX_DUAL:
      e = launch_prefix_dual(p, plan->lay.max_rows, q, k_prefix, v_prefix, plan->total_prefix_tokens, k_pool,
                             v_pool, !timed, s);
      break;
    default: return fail(PAD_ERR_UNSUPPORTED, "prefix kernel %d", plan->lay.prefix_kernel);
  }
  if (e != cudaSuccess) return cuda_fail(e, "prefix launch");
  if (timed) {
    cudaEventRecord(g_timing.ev[2 * g_timing.n + 1], s);
    g_timing.n++;
  }
  if (!plan->lay.fused) {
    const bool pdl = !timed && (plan->lay.prefix_kernel == PAD_FLAG_PREFIX_TC ||
                                plan->lay.prefix_kernel == PAD_FLAG_PREFIX_DUAL);
    e = launch_branch_merge(p, q, k_pool, v_pool, out, lse, pdl, s);
    if (e != cudaSuccess) return cuda_fail(e, "branch/merge launch");
  }
  if (plan->image) {
    e = cudaEventRecord(plan->image->done, s);
    if (e != cudaSuccess) return cuda_fail(e, "plan image event");
    plan->image->recorded = true;
  }
  return PAD_OK;
}

pad_status pad_event_decode_attn(const pad_plan_t* plan, const void* q, const void* k_prefix,
                                 const void* v_prefix, const void* k_pool, const void* v_pool,
                                 void* out, float* lse, pad_stream_t stream) {
  NvtxRange nvtx_range("pad_event_decode_attn");
  return launch_attention(plan, q, nullptr, nullptr, k_prefix, v_prefix, k_pool, v_pool, out, lse, stream);
}

pad_status pad_decode_step(const pad_plan_t* plan, const void* q, const void* k_new, const void* v_new,
                           const void* k_prefix, const void* v_prefix, void* k_pool, void* v_pool,
                           void* out, float* lse, pad_stream_t stream) {
  NvtxRange nvtx_range("pad_decode_step");
  if (plan && plan->n_events > 0 && (!k_new || !v_new)) return fail(PAD_ERR_INVALID_ARG, "NULL k_new / v_new");
  return launch_attention(plan, q, k_new, v_new, k_prefix, v_prefix, k_pool, v_pool, out, lse, stream);
}

// ---------------------------------------------------------------------------
// Step executor: a serving loop's host side in one call per step.
// ---------------------------------------------------------------------------
struct pad_step_t {
  pad_problem prob{};
  pad_cache_state* cache = nullptr;
  int32_t n_videos = 0, n_events = 0, max_pages = 0, options = 0;
  const int32_t* prefix_len = nullptr;
  const int64_t* prefix_offset = nullptr;
  const int32_t* event_video = nullptr;
  const int32_t* event_len = nullptr;
  int32_t* page_table = nullptr;
  void* workspace = nullptr;
  size_t workspace_bytes = 0;
  const void *q = nullptr, *k_new = nullptr, *v_new = nullptr, *k_prefix = nullptr, *v_prefix = nullptr;
  void *k_pool = nullptr, *v_pool = nullptr, *out = nullptr;
  float* lse = nullptr;
  pad_stream_t stream = nullptr;
  const int32_t* rope_pos = nullptr;
  const float* rope_cs = nullptr;
  int32_t rope_max = 0;
  int32_t g_mode = PAD_G_ALL;
  const int32_t* g_planning = nullptr;
  const int32_t* g_index = nullptr;
  int32_t branch_mode = PAD_BRANCH_OWN;
  // pad_step_profile: CUDA events between the phases of pad_step_run_host and host clock
  // readings around them, summed over the profiled calls
  struct Profile {
    bool on = false;
    cudaEvent_t ev[5] = {};
    int64_t n = 0;
    double host[6] = {};  // input copy call, pad_plan, launches, output copy call, wait, total
    double dev[5] = {};   // input copy, wait for the plan, kernels, output copy, whole span
  } prof;
  // pad_step_enqueue_host: recorded behind the latest enqueued run, waited on by pad_step_wait
  cudaEvent_t done = nullptr;
  bool pending = false;
  ~pad_step_t() {
    for (cudaEvent_t& e : prof.ev)
      if (e) cudaEventDestroy(e);
    if (done) cudaEventDestroy(done);
  }
};

namespace {
double host_us() {
  return std::chrono::duration<double, std::micro>(std::chrono::steady_clock::now().time_since_epoch()).count();
}
}  // namespace

pad_status pad_step_create(const pad_problem* prob, pad_cache_state* cache, int32_t n_videos,
                           const int32_t* prefix_len, const int64_t* prefix_offset, int32_t n_events,
                           const int32_t* event_video, const int32_t* event_len, int32_t* page_table,
                           int32_t max_pages, void* workspace, size_t workspace_bytes, const void* q,
                           const void* k_new, const void* v_new, const void* k_prefix, const void* v_prefix,
                           void* k_pool, void* v_pool, void* out, float* lse, pad_stream_t stream,
                           int32_t options, pad_step_t** step_out) {
  if (!step_out) return fail(PAD_ERR_INVALID_ARG, "step_out is NULL");
  *step_out = nullptr;
  pad_status st = check_problem(prob);
  if (st != PAD_OK) return st;
  if (!cache) return fail(PAD_ERR_INVALID_ARG, "cache is NULL");
  if (options & ~(PAD_STEP_TWO_CALL | PAD_STEP_RELEASE_PAGES | PAD_STEP_MAPPED_HOST_IO))
    return fail(PAD_ERR_INVALID_ARG, "unknown options 0x%x", options);
  if (n_videos < 0 || n_events < 0) return fail(PAD_ERR_INVALID_ARG, "negative batch size");
  if (n_events > 0 && (!event_video || !event_len || !prefix_len)) return fail(PAD_ERR_INVALID_ARG, "NULL host array");
  if (!workspace || !page_table) return fail(PAD_ERR_INVALID_ARG, "workspace / page_table is NULL");
  if (n_events > 0 && (!q || !k_pool || !v_pool || !out || !k_new || !v_new))
    return fail(PAD_ERR_INVALID_ARG, "NULL tensor");
  auto* x = new pad_step_t();
  x->prob = *prob;
  x->cache = cache;
  x->n_videos = n_videos;
  x->n_events = n_events;
  x->max_pages = max_pages;
  x->options = options;
  x->prefix_len = prefix_len;
  x->prefix_offset = prefix_offset;
  x->event_video = event_video;
  x->event_len = event_len;
  x->page_table = page_table;
  x->workspace = workspace;
  x->workspace_bytes = workspace_bytes;
  x->q = q;
  x->k_new = k_new;
  x->v_new = v_new;
  x->k_prefix = k_prefix;
  x->v_prefix = v_prefix;
  x->k_pool = k_pool;
  x->v_pool = v_pool;
  x->out = out;
  x->lse = lse;
  x->stream = stream;
  *step_out = x;
  return PAD_OK;
}

pad_status pad_step_set_rope(pad_step_t* step, const int32_t* positions, const float* cos_sin, int32_t max_position) {
  if (!step) return fail(PAD_ERR_INVALID_ARG, "step is NULL");
  if (cos_sin && (max_position <= 0 || !aligned16(cos_sin) || (step->n_events > 0 && !positions)))
    return fail(PAD_ERR_INVALID_ARG, "positions / cos_sin / max_position");
  step->rope_pos = cos_sin ? positions : nullptr;
  step->rope_cs = cos_sin;
  step->rope_max = cos_sin ? max_position : 0;
  return PAD_OK;
}

pad_status pad_step_set_g_visibility(pad_step_t* step, int32_t mode, const int32_t* n_planning,
                                     const int32_t* g_index) {
  if (!step) return fail(PAD_ERR_INVALID_ARG, "step is NULL");
  if (mode != PAD_G_ALL && mode != PAD_G_SELF) return fail(PAD_ERR_INVALID_ARG, "mode %d", mode);
  if (mode == PAD_G_SELF && ((step->n_videos > 0 && !n_planning) || (step->n_events > 0 && !g_index)))
    return fail(PAD_ERR_INVALID_ARG, "n_planning / g_index is NULL");
  step->g_mode = mode;
  step->g_planning = n_planning;
  step->g_index = g_index;
  return PAD_OK;
}

pad_status pad_step_set_branch_visibility(pad_step_t* step, int32_t mode) {
  if (!step) return fail(PAD_ERR_INVALID_ARG, "step is NULL");
  if (mode != PAD_BRANCH_OWN && mode != PAD_BRANCH_CAUSAL) return fail(PAD_ERR_INVALID_ARG, "mode %d", mode);
  step->branch_mode = mode;
  return PAD_OK;
}

namespace {
// One step: pad_plan, the launches (writing O and LSE to `out` / `lse`), page bookkeeping.
// With `ht` (profiling) it records event 2 and host time 2 after planning, event 3 and host
// time 3 after the launches.
pad_status step_run(pad_step_t* step, int32_t* new_page, double* ht, void* out, float* lse) {
  pad_plan_t* plan = nullptr;
  pad_status st = pad_plan(&step->prob, step->cache, step->n_videos, step->prefix_len, step->prefix_offset,
                           step->n_events, step->event_video, step->event_len, step->page_table, step->max_pages,
                           step->workspace, step->workspace_bytes, step->stream, &plan);
  if (st != PAD_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(step->stream);
  if (ht) {
    ht[2] = host_us();
    cudaEventRecord(step->prof.ev[2], s);
  }
  if (step->rope_cs) st = pad_plan_set_rope(plan, step->rope_pos, step->rope_cs, step->rope_max);
  if (st == PAD_OK && step->g_mode == PAD_G_SELF)
    st = pad_plan_set_g_visibility(plan, PAD_G_SELF, step->g_planning, step->g_index);
  if (st == PAD_OK && step->branch_mode == PAD_BRANCH_CAUSAL) st = pad_plan_set_branch_visibility(plan, PAD_BRANCH_CAUSAL);
  bool wrote_pages = false;  // the append kernel has been launched: the pages are in the table
  if (st == PAD_OK) {
    if (step->options & PAD_STEP_TWO_CALL) {
      st = pad_kv_append(plan, step->k_new, step->v_new, step->k_pool, step->v_pool, step->stream);
      wrote_pages = st == PAD_OK;
      if (st == PAD_OK)
        st = pad_event_decode_attn(plan, step->q, step->k_prefix, step->v_prefix, step->k_pool, step->v_pool,
                                   out, lse, step->stream);
    } else {
      st = pad_decode_step(plan, step->q, step->k_new, step->v_new, step->k_prefix, step->v_prefix, step->k_pool,
                           step->v_pool, out, lse, step->stream);
    }
  }
  if (ht) {
    ht[3] = host_us();
    cudaEventRecord(step->prof.ev[3], s);
  }
  if (st == PAD_OK && new_page) st = pad_plan_new_pages(plan, new_page);
  if ((st != PAD_OK && !wrote_pages) || (step->options & PAD_STEP_RELEASE_PAGES)) {
    // a step that failed before any kernel wrote its pages into the table hands them back
    // (in the one-call step the branch/merge kernel writes them, and it is launched last);
    // so does a timing loop
    const pad_status keep = st;
    pad_plan_release_new_pages(plan, step->cache);
    st = keep;
  }
  pad_plan_destroy(plan);
  return st;
}
}  // namespace

pad_status pad_step_run(pad_step_t* step, int32_t* new_page) {
  NvtxRange nvtx_range("pad_step_run");
  if (!step) return fail(PAD_ERR_INVALID_ARG, "step is NULL");
  return step_run(step, new_page, nullptr, step->out, step->lse);
}

pad_status pad_step_profile(pad_step_t* step, int32_t enable) {
  if (!step) return fail(PAD_ERR_INVALID_ARG, "step is NULL");
  auto& pr = step->prof;
  if (enable) {
    for (cudaEvent_t& e : pr.ev) {
      if (e) continue;
      cudaError_t ce = cudaEventCreate(&e);
      if (ce != cudaSuccess) return cuda_fail(ce, "cudaEventCreate");
    }
  }
  pr.on = enable != 0;
  pr.n = 0;
  for (double& v : pr.host) v = 0.0;
  for (double& v : pr.dev) v = 0.0;
  return PAD_OK;
}

pad_status pad_step_profile_read(const pad_step_t* step, double* out, int32_t n) {
  if (!step || !out) return fail(PAD_ERR_INVALID_ARG, "NULL argument");
  if (n < 12) return fail(PAD_ERR_INVALID_ARG, "out needs 12 entries; got %d", n);
  const auto& pr = step->prof;
  const double c = pr.n > 0 ? 1.0 / (double)pr.n : 0.0;
  out[0] = (double)pr.n;
  for (int i = 0; i < 6; ++i) out[1 + i] = pr.host[i] * c;
  for (int i = 0; i < 5; ++i) out[7 + i] = pr.dev[i] * c;
  return PAD_OK;
}

namespace {
// Device address of host range [h, h + n) when it is page-locked, device-mapped memory
// (checked at its first and last byte, which must map n - 1 bytes apart) and aligned to
// `align` bytes; nullptr otherwise.
void* mapped_view(const void* h, size_t n, size_t align) {
  if (!h || n == 0 || (reinterpret_cast<uintptr_t>(h) % align) != 0) return nullptr;
  cudaPointerAttributes a0{}, a1{};
  if (cudaPointerGetAttributes(&a0, h) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  const char* last = static_cast<const char*>(h) + (n - 1);
  if (cudaPointerGetAttributes(&a1, last) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  if (a0.type != cudaMemoryTypeHost || a1.type != cudaMemoryTypeHost || !a0.devicePointer || !a1.devicePointer)
    return nullptr;
  if (static_cast<const char*>(a1.devicePointer) - static_cast<const char*>(a0.devicePointer) != (ptrdiff_t)(n - 1))
    return nullptr;
  return a0.devicePointer;
}
}  // namespace

namespace {
// pad_step_run_host (wait) and pad_step_enqueue_host (no wait: an event behind the run)
pad_status host_step(pad_step_t* step, const void* h_q, const void* h_k_new, const void* h_v_new, void* h_out,
                     float* h_lse, int32_t* new_page, bool wait) {
  NvtxRange nvtx_range(wait ? "pad_step_run_host" : "pad_step_enqueue_host");
  if (!step) return fail(PAD_ERR_INVALID_ARG, "step is NULL");
  if (step->n_events > 0 && (!h_q || !h_k_new || !h_v_new || !h_out))
    return fail(PAD_ERR_INVALID_ARG, "NULL host buffer");
  if (step->n_events > 0 && h_lse && !step->lse) return fail(PAD_ERR_INVALID_ARG, "h_lse given but the step has no lse");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(step->stream);
  const pad_problem& pr = step->prob;
  const size_t E = (size_t)step->n_events, D = (size_t)pr.head_dim;
  const size_t q_bytes = E * pr.h_q * D * 2, kv_bytes = E * pr.h_kv * D * 2;
  const size_t o_bytes = E * pr.h_q * D * (pr.out_dtype == 1 ? 2 : 4), l_bytes = E * pr.h_q * sizeof(float);
  // buffers that follow one another in device memory and in host memory alike go in one copy
  auto adjacent = [](const void* a, size_t n, const void* b) {
    return static_cast<const char*>(a) + n == static_cast<const char*>(b);
  };
  cudaError_t e = cudaSuccess;
  auto& prof = step->prof;
  double ht[6] = {};
  double* htp = (prof.on && wait) ? ht : nullptr;
  if (!wait && !step->done) {
    e = cudaEventCreateWithFlags(&step->done, cudaEventDisableTiming);
    if (e != cudaSuccess) return cuda_fail(e, "cudaEventCreate");
  }
  if (htp) {
    ht[0] = host_us();
    cudaEventRecord(prof.ev[0], s);
  }
  // mapped host I/O: device views of every host buffer, else the copy path
  void *vq = nullptr, *vk = nullptr, *vv = nullptr, *vo = nullptr, *vl = nullptr;
  bool mapped = false;
  if (E > 0 && (step->options & PAD_STEP_MAPPED_HOST_IO)) {
    vq = mapped_view(h_q, q_bytes, 16);
    vk = vq ? mapped_view(h_k_new, kv_bytes, 16) : nullptr;
    vv = vk ? mapped_view(h_v_new, kv_bytes, 16) : nullptr;
    vo = vv ? mapped_view(h_out, o_bytes, 16) : nullptr;
    vl = (vo && h_lse) ? mapped_view(h_lse, l_bytes, 4) : nullptr;
    mapped = vo && (!h_lse || vl) && aligned16(step->q) && aligned16(step->k_new) && aligned16(step->v_new);
  }
  if (mapped) {
    const void* src[3];
    void* dst[3];
    size_t nb[3];
    int n = 0;
    const bool kq = adjacent(step->q, q_bytes, step->k_new) && adjacent(vq, q_bytes, vk);
    const bool vk_adj = adjacent(step->k_new, kv_bytes, step->v_new) && adjacent(vk, kv_bytes, vv);
    if (kq && vk_adj) {
      src[n] = vq, dst[n] = const_cast<void*>(step->q), nb[n++] = q_bytes + 2 * kv_bytes;
    } else {
      src[n] = vq, dst[n] = const_cast<void*>(step->q), nb[n++] = q_bytes;
      src[n] = vk, dst[n] = const_cast<void*>(step->k_new), nb[n++] = kv_bytes;
      src[n] = vv, dst[n] = const_cast<void*>(step->v_new), nb[n++] = kv_bytes;
    }
    e = launch_host_in(src, dst, nb, n, query_num_sms(), s);
    if (e != cudaSuccess) {
      cudaStreamSynchronize(s);
      return cuda_fail(e, "step inputs from mapped host memory");
    }
  } else if (E > 0) {
    char* dq = static_cast<char*>(const_cast<void*>(step->q));
    const char* hq = static_cast<const char*>(h_q);
    const bool kq = adjacent(step->q, q_bytes, step->k_new) && adjacent(h_q, q_bytes, h_k_new);
    const bool vk = adjacent(step->k_new, kv_bytes, step->v_new) && adjacent(h_k_new, kv_bytes, h_v_new);
    if (kq && vk) {
      e = cudaMemcpyAsync(dq, hq, q_bytes + 2 * kv_bytes, cudaMemcpyHostToDevice, s);
    } else {
      e = cudaMemcpyAsync(dq, hq, q_bytes, cudaMemcpyHostToDevice, s);
      if (e == cudaSuccess) e = cudaMemcpyAsync(const_cast<void*>(step->k_new), h_k_new, kv_bytes, cudaMemcpyHostToDevice, s);
      if (e == cudaSuccess) e = cudaMemcpyAsync(const_cast<void*>(step->v_new), h_v_new, kv_bytes, cudaMemcpyHostToDevice, s);
    }
    if (e != cudaSuccess) {
      cudaStreamSynchronize(s);  // the host buffers are the caller's again when this returns
      return cuda_fail(e, "step inputs H2D");
    }
  }
  if (htp) {
    ht[1] = host_us();
    cudaEventRecord(prof.ev[1], s);
  }
  pad_status st = mapped ? step_run(step, new_page, htp, vo, static_cast<float*>(vl))
                         : step_run(step, new_page, htp, step->out, step->lse);
  if (st != PAD_OK) {
    const std::string msg = g_last_error;
    cudaStreamSynchronize(s);
    g_last_error = msg;
    return st;
  }
  if (E > 0 && !mapped) {
    if (h_lse && adjacent(step->out, o_bytes, step->lse) && adjacent(h_out, o_bytes, h_lse)) {
      e = cudaMemcpyAsync(h_out, step->out, o_bytes + l_bytes, cudaMemcpyDeviceToHost, s);
    } else {
      e = cudaMemcpyAsync(h_out, step->out, o_bytes, cudaMemcpyDeviceToHost, s);
      if (e == cudaSuccess && h_lse) e = cudaMemcpyAsync(h_lse, step->lse, l_bytes, cudaMemcpyDeviceToHost, s);
    }
    if (e != cudaSuccess) {
      cudaStreamSynchronize(s);
      return cuda_fail(e, "step outputs D2H");
    }
  }
  if (!wait) {
    e = cudaEventRecord(step->done, s);
    if (e != cudaSuccess) {
      cudaStreamSynchronize(s);
      return cuda_fail(e, "cudaEventRecord");
    }
    step->pending = true;
    return PAD_OK;
  }
  if (htp) {
    ht[4] = host_us();
    cudaEventRecord(prof.ev[4], s);
  }
  e = cudaStreamSynchronize(s);
  if (e == cudaSuccess && htp) {
    ht[5] = host_us();
    const double hd[6] = {ht[1] - ht[0], ht[2] - ht[1], ht[3] - ht[2], ht[4] - ht[3], ht[5] - ht[4], ht[5] - ht[0]};
    float dv[5] = {};
    for (int i = 0; i < 4; ++i) cudaEventElapsedTime(&dv[i], prof.ev[i], prof.ev[i + 1]);
    cudaEventElapsedTime(&dv[4], prof.ev[0], prof.ev[4]);
    for (int i = 0; i < 6; ++i) prof.host[i] += hd[i];
    for (int i = 0; i < 5; ++i) prof.dev[i] += 1e3 * (double)dv[i];
    ++prof.n;
  }
  step->pending = false;
  return e == cudaSuccess ? PAD_OK : cuda_fail(e, "step synchronize");
}
}  // namespace

pad_status pad_step_run_host(pad_step_t* step, const void* h_q, const void* h_k_new, const void* h_v_new,
                             void* h_out, float* h_lse, int32_t* new_page) {
  return host_step(step, h_q, h_k_new, h_v_new, h_out, h_lse, new_page, true);
}

pad_status pad_step_enqueue_host(pad_step_t* step, const void* h_q, const void* h_k_new, const void* h_v_new,
                                 void* h_out, float* h_lse, int32_t* new_page) {
  return host_step(step, h_q, h_k_new, h_v_new, h_out, h_lse, new_page, false);
}

pad_status pad_step_wait(pad_step_t* step) {
  if (!step) return fail(PAD_ERR_INVALID_ARG, "step is NULL");
  if (!step->pending) return PAD_OK;
  step->pending = false;
  const cudaError_t e = cudaEventSynchronize(step->done);
  return e == cudaSuccess ? PAD_OK : cuda_fail(e, "step wait");
}

void pad_step_destroy(pad_step_t* step) { delete step; }

pad_status pad_device_status(const pad_plan_t* plan, pad_stream_t stream) {
  if (!plan) return fail(PAD_ERR_INVALID_ARG, "plan is NULL");
  // a host-only plan reports through the static scratch array's status word (if no call
  // has used the array on this device, nothing of this plan ran there)
  const void* word = plan->workspace;
  if (!word) {
    PadDevHeader* sh = nullptr;
    pad_status st = static_status_header(&sh);
    if (st != PAD_OK) return st;
    if (!sh) return PAD_OK;
    word = sh;
  }
  PadDevHeader h;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e = cudaMemcpyAsync(&h, word, sizeof(h), cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(e, "reading device status");
  const int code = (int)(h.word & 0xffull);
  if ((h.word >> 8) == plan->gen && code != PAD_OK) {
    // a failed launch may have left the fused tail's split counters part-way: zero them,
    // so that the next plan on this workspace starts clean
    if (plan->lay.n_counters > 0 && plan->workspace) {
      e = cudaMemsetAsync(static_cast<uint8_t*>(plan->workspace) + plan->lay.off_cnt, 0,
                          (size_t)plan->lay.n_counters * sizeof(unsigned int), s);
      if (e == cudaSuccess) e = cudaStreamSynchronize(s);
      if (e != cudaSuccess) return cuda_fail(e, "clearing split counters");
    }
    return fail((pad_status)code, "device reported %s (detail %d %d %d)",
                pad_status_string((pad_status)code), h.info[0], h.info[1], h.info[2]);
  }
  return PAD_OK;
}

pad_status pad_timing_enable(int32_t max_launches) {
  if (max_launches <= 0) return fail(PAD_ERR_INVALID_ARG, "max_launches must be > 0");
  while ((int)g_timing.ev.size() < 2 * max_launches) {
    cudaEvent_t ev;
    cudaError_t e = cudaEventCreate(&ev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaEventCreate");
    g_timing.ev.push_back(ev);
  }
  g_timing.on = true;
  g_timing.max = max_launches;
  g_timing.n = 0;
  return PAD_OK;
}

pad_status pad_timing_read(float* total_ms, int32_t* n_launches) {
  if (!total_ms || !n_launches) return fail(PAD_ERR_INVALID_ARG, "NULL argument");
  float tot = 0.f;
  for (int i = 0; i < g_timing.n; ++i) {
    cudaError_t e = cudaEventSynchronize(g_timing.ev[2 * i + 1]);
    if (e != cudaSuccess) return cuda_fail(e, "cudaEventSynchronize");
    float ms = 0.f;
    e = cudaEventElapsedTime(&ms, g_timing.ev[2 * i], g_timing.ev[2 * i + 1]);
    if (e != cudaSuccess) return cuda_fail(e, "cudaEventElapsedTime");
    tot += ms;
  }
  *total_ms = tot;
  *n_launches = g_timing.n;
  g_timing.on = false;
  g_timing.n = 0;
  return PAD_OK;
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Allocation-free variant of pad_event_decode_attn.
//
// Some callers have no way to hand this library device memory for scratch: a host
// application's plugin interface that gives out tensors but no allocator, a serving
// loop whose memory is reserved up front and must not grow or fragment while it
// runs, or a process whose device memory is owned by an allocator it cannot call
// into.  For them the plan image and the split-KV partial states live in the array
// below instead of a caller workspace; the caller still passes every input and output.
//
// The array is a file-scope device variable: every GPU that loads this library keeps
// kStaticScratchBytes of device memory for it until the process exits.  Its device
// address is fetched once per device (cudaGetSymbolAddress on the first call made with
// that device current) and cached.  All calls share the array, so two calls whose work
// overlaps on the GPU (different streams, or different host threads) race on it; calls
// ordered on one stream are safe, each one re-uploading the plan image, which also
// clears the status word.
// ---------------------------------------------------------------------------
namespace {

constexpr size_t kStaticScratchBytes = 16u << 20;  // 16 MiB
static __device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

std::mutex g_static_mu;
void* g_static_ptr[64] = {};

// The static array's device address on the current device, looked up on the first call
// made with that device current and cached (lookup = false: only the cached address, or
// NULL when no call has used the array on this device yet).
pad_status static_scratch(bool lookup, uint8_t** out) {
  *out = nullptr;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (dev < 0 || dev >= 64) return fail(PAD_ERR_UNSUPPORTED, "device index %d", dev);
  std::lock_guard<std::mutex> lk(g_static_mu);
  if (!g_static_ptr[dev] && lookup) {
    void* ptr = nullptr;
    e = cudaGetSymbolAddress(&ptr, g_static_scratch);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(static scratch)");
    g_static_ptr[dev] = ptr;
  }
  *out = static_cast<uint8_t*>(g_static_ptr[dev]);
  return PAD_OK;
}

// Launch parameters of a plan whose scratch is the static array.  The plan image (video
// and event descriptors, work items) is copied into the array on `s`, from the plan's own
// pageable host buffer: the driver stages that copy, so the call returns once the bytes
// are staged.  The status word ahead of the image is left as it is: it is tagged with the
// generation of the plan whose kernels wrote it, so a word from another plan reads as
// clear, and an error of this plan's append survives until its attention call and
// pad_device_status read it.
pad_status static_params(const pad_plan_t* plan, cudaStream_t s, KParams& p, uint8_t** ws_out) {
  if (plan->lay.total_bytes > kStaticScratchBytes)
    return fail(PAD_ERR_WORKSPACE_TOO_SMALL,
                "plan needs %zu bytes of scratch; the static scratch array holds %zu bytes",
                plan->lay.total_bytes, kStaticScratchBytes);
  uint8_t* ws = nullptr;
  pad_status st = static_scratch(true, &ws);
  if (st != PAD_OK) return st;
  const size_t hb = sizeof(PadDevHeader);
  if (plan->lay.upload_bytes > hb) {
    cudaError_t e = cudaMemcpyAsync(ws + hb, plan->host_image.data() + hb, plan->lay.upload_bytes - hb,
                                    cudaMemcpyHostToDevice, s);
    if (e != cudaSuccess) return cuda_fail(e, "static scratch plan upload");
  }
  const pad_problem& pr = plan->prob;
  p.h_q = pr.h_q;
  p.h_kv = pr.h_kv;
  p.group = pr.h_q / pr.h_kv;
  p.head_dim = pr.head_dim;
  p.page_size = pr.page_size;
  p.max_pages = plan->max_pages;
  p.n_pages = plan->n_pages;
  p.n_videos = plan->n_videos;
  p.n_events = plan->n_events;
  p.n_items = (int32_t)plan->lay.n_items;
  p.out_bf16 = pr.out_dtype == 1;
  p.n_sms = plan->lay.n_sms;
  p.max_splits = 0;
  for (int32_t ns : plan->lay.n_splits) p.max_splits = std::max(p.max_splits, ns);
  p.branch_rows = std::min(128, ((plan->causal ? plan->task_keys : plan->max_event_len + 1) + 15) / 16 * 16);
  p.scale_log2 = (float)((double)pr.scale * 1.4426950408889634);
  p.gen = plan->gen;
  p.img_n = 0;
  p.k_new = nullptr;
  p.v_new = nullptr;
  p.rope_cs = plan->rope_cs;
  p.g_self = plan->g_self;
  p.causal = plan->causal;
  p.fused = plan->lay.fused ? 1 : 0;
  p.cta_map = plan->lay.cta_map ? 1 : 0;
  p.n_ctas = (int32_t)plan->lay.n_ctas;
  p.tail_chunk = p.fused ? prefix_tc_tail_chunk(p.branch_rows, p.group, p.max_splits) : 0;
  p.merge_first = plan->lay.merge_first ? 1 : 0;
  p.tasks = reinterpret_cast<const int32_t*>(ws + plan->lay.off_tasks);
  p.counters = reinterpret_cast<unsigned int*>(ws + plan->lay.off_cnt);
  p.n_counters = p.fused ? (int32_t)plan->lay.n_counters : 0;
  p.header = reinterpret_cast<PadDevHeader*>(ws);
  p.videos = reinterpret_cast<const PadVideoDesc*>(ws + plan->lay.off_videos);
  p.events = reinterpret_cast<const PadEventDesc*>(ws + plan->lay.off_events);
  p.items = reinterpret_cast<const PadWorkItem*>(ws + plan->lay.off_items);
  p.part_ml = reinterpret_cast<float2*>(ws + plan->lay.off_ml);
  p.part_o = reinterpret_cast<float*>(ws + plan->lay.off_o);
  p.page_table = plan->page_table;
  *ws_out = ws;
  return PAD_OK;
}

}  // namespace

// pad_kv_append of a plan built without a workspace: the append kernel reads the plan's
// event descriptors from the static array and reports into its status word.
static pad_status static_kv_append(const pad_plan_t* plan, const void* k_new, const void* v_new, void* k_pool,
                                   void* v_pool, cudaStream_t s) {
  KParams p;
  uint8_t* ws = nullptr;
  pad_status st = static_params(plan, s, p, &ws);
  if (st != PAD_OK) return st;
  cudaError_t e = launch_append(p, k_new, v_new, k_pool, v_pool, s);
  if (e != cudaSuccess) return cuda_fail(e, "append launch (static scratch)");
  return PAD_OK;
}

// The static array's status header, or NULL when no call has used the array on the
// current device.
static pad_status static_status_header(PadDevHeader** out) {
  uint8_t* ws = nullptr;
  pad_status st = static_scratch(false, &ws);
  *out = reinterpret_cast<PadDevHeader*>(ws);
  return st;
}

extern "C" pad_status pad_event_decode_attn_static(const pad_plan_t* plan, const void* q,
                                                   const void* k_prefix, const void* v_prefix,
                                                   const void* k_pool, const void* v_pool, void* out,
                                                   float* lse, pad_stream_t stream) {
  if (!plan) return fail(PAD_ERR_INVALID_ARG, "plan is NULL");
  if (plan->n_events == 0) return PAD_OK;
  if (plan->lay.total_bytes > kStaticScratchBytes)
    return fail(PAD_ERR_WORKSPACE_TOO_SMALL,
                "plan needs %zu bytes of scratch; the static scratch array holds %zu bytes",
                plan->lay.total_bytes, kStaticScratchBytes);
  if (!plan->page_table) return fail(PAD_ERR_INVALID_ARG, "plan has no page table");
  if (!q || !k_pool || !v_pool || !out) return fail(PAD_ERR_INVALID_ARG, "NULL tensor");
  if (plan->lay.n_items > 0 && (!k_prefix || !v_prefix))
    return fail(PAD_ERR_INVALID_ARG, "k_prefix / v_prefix is NULL");
  if (!aligned16(q) || !aligned16(k_prefix) || !aligned16(v_prefix) || !aligned16(k_pool) ||
      !aligned16(v_pool) || !aligned16(out) || (lse && (reinterpret_cast<uintptr_t>(lse) & 3u)))
    return fail(PAD_ERR_INVALID_ARG, "tensors must be 16-byte aligned (lse 4-byte)");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  KParams p;
  uint8_t* ws = nullptr;
  pad_status st = static_params(plan, s, p, &ws);
  if (st != PAD_OK) return st;
  cudaError_t e = cudaSuccess;
  switch (plan->lay.prefix_kernel) {
    case PAD_FLAG_PREFIX_SIMT: e = launch_prefix_simt(p, plan->lay.max_rows, q, k_prefix, v_prefix, s); break;
    case PAD_FLAG_PREFIX_MMA: e = launch_prefix_mma(p, plan->lay.max_rows, q, k_prefix, v_prefix, s); break;
    case PAD_FLAG_PREFIX_TC:
      if (p.n_counters > 0) {  // (the append of a workspace plan zeroes them; none ran on this array)
        e = cudaMemsetAsync(ws + plan->lay.off_cnt, 0, (size_t)p.n_counters * sizeof(unsigned int), s);
        if (e != cudaSuccess) return cuda_fail(e, "static scratch counters");
      }
      e = launch_prefix_tc(p, plan->lay.max_rows, q, k_prefix, v_prefix, plan->total_prefix_tokens, k_pool,
                           v_pool, out, lse, false, s);
      break;
    case PAD_FLAG_PREFIX_DUAL:
      e = launch_prefix_dual(p, plan->lay.max_rows, q, k_prefix, v_prefix, plan->total_prefix_tokens, k_pool,
                             v_pool, false, s);
      break;
    default: return fail(PAD_ERR_UNSUPPORTED, "prefix kernel %d", plan->lay.prefix_kernel);
  }
  if (e != cudaSuccess) return cuda_fail(e, "prefix launch (static scratch)");
  if (!plan->lay.fused) {
    e = launch_branch_merge(p, q, k_pool, v_pool, out, lse, false, s);
    if (e != cudaSuccess) return cuda_fail(e, "branch/merge launch (static scratch)");
  }
  return PAD_OK;
}

// ---------------------------------------------------------------------------
// Grounding readout (Sec. 3.3)
// ---------------------------------------------------------------------------

static pad_status check_offsets(const int32_t* offsets, int32_t n_segments, int64_t n_tokens) {
  if (n_segments < 1 || n_segments > 1024) return fail(PAD_ERR_UNSUPPORTED, "n_segments=%d outside [1, 1024]", n_segments);
  if (!offsets) return fail(PAD_ERR_INVALID_ARG, "offsets is NULL");
  for (int s = 0; s <= n_segments; ++s)
    if (offsets[s] < 0 || offsets[s] > n_tokens || (s > 0 && offsets[s] < offsets[s - 1]))
      return fail(PAD_ERR_INVALID_ARG, "offsets[%d]=%d: must be non-decreasing within [0, %lld]", s, offsets[s],
                  (long long)n_tokens);
  return PAD_OK;
}

pad_status pad_ground_pool(const void* f_proj, int64_t n_tokens, int32_t d_proj, const int32_t* offsets,
                           int32_t n_segments, float* seg_sum, pad_stream_t stream) {
  if (d_proj < 8 || d_proj > 2048 || d_proj % 8) return fail(PAD_ERR_UNSUPPORTED, "d_proj=%d: a multiple of 8 up to 2048", d_proj);
  if (n_tokens < 0 || n_tokens > INT32_MAX) return fail(PAD_ERR_INVALID_ARG, "n_tokens=%lld", (long long)n_tokens);
  pad_status st = check_offsets(offsets, n_segments, n_tokens);
  if (st != PAD_OK) return st;
  if (!f_proj || !seg_sum) return fail(PAD_ERR_INVALID_ARG, "NULL tensor");
  if (!aligned16(f_proj) || !aligned16(seg_sum)) return fail(PAD_ERR_INVALID_ARG, "tensors must be 16-byte aligned");
  cudaError_t e = launch_ground_pool(f_proj, n_tokens, d_proj, offsets, n_segments, seg_sum,
                                     reinterpret_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? PAD_OK : cuda_fail(e, "ground pool launch");
}

pad_status pad_ground_score(const void* g_proj, int32_t n_events, const float* seg_sum, int32_t n_segments,
                            int32_t d_proj, float fraction, float* scores, uint8_t* salient, int32_t* interval,
                            pad_stream_t stream) {
  if (d_proj < 8 || d_proj > 2048 || d_proj % 8) return fail(PAD_ERR_UNSUPPORTED, "d_proj=%d: a multiple of 8 up to 2048", d_proj);
  if (n_segments < 1 || n_segments > 1024) return fail(PAD_ERR_UNSUPPORTED, "n_segments=%d outside [1, 1024]", n_segments);
  if (n_events < 0) return fail(PAD_ERR_INVALID_ARG, "n_events < 0");
  if (!(fraction >= 0.f && fraction <= 1.f)) return fail(PAD_ERR_INVALID_ARG, "fraction must be in [0, 1]");
  if (n_events > 0 && (!g_proj || !seg_sum || !scores || !salient || !interval)) return fail(PAD_ERR_INVALID_ARG, "NULL tensor");
  if (!aligned16(g_proj) || !aligned16(seg_sum)) return fail(PAD_ERR_INVALID_ARG, "tensors must be 16-byte aligned");
  cudaError_t e = launch_ground_score(g_proj, n_events, seg_sum, n_segments, d_proj, fraction, scores, salient,
                                      interval, reinterpret_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? PAD_OK : cuda_fail(e, "ground score launch");
}

size_t pad_attn_aggregate_workspace_size(int64_t n_tokens, int32_t n_segments, int32_t d_model) {
  if (n_tokens < 0 || n_segments < 1 || d_model < 1) return 0;
  return attn_aggregate_ws_floats(n_tokens, n_segments, d_model) * sizeof(float);
}

pad_status pad_attn_aggregate(const void* x, int64_t n_tokens, int32_t d_model, const float* attn,
                              const int32_t* offsets, int32_t n_segments, const int32_t* interval, int32_t n_events,
                              const void* g_emb, float* seg_ws, size_t seg_ws_bytes, float* out,
                              pad_stream_t stream) {
  if (d_model < 8 || d_model % 8 || d_model > (1 << 24)) return fail(PAD_ERR_UNSUPPORTED, "d_model=%d: a multiple of 8", d_model);
  if (n_tokens < 0 || n_tokens > INT32_MAX) return fail(PAD_ERR_INVALID_ARG, "n_tokens=%lld", (long long)n_tokens);
  pad_status st = check_offsets(offsets, n_segments, n_tokens);
  if (st != PAD_OK) return st;
  if (n_events < 0 || n_events > 65535) return fail(PAD_ERR_INVALID_ARG, "n_events=%d", n_events);
  if (n_events > 0 && (!x || !attn || !interval || !g_emb || !seg_ws || !out))
    return fail(PAD_ERR_INVALID_ARG, "NULL tensor");
  if (!aligned16(x) || !aligned16(g_emb) || !aligned16(seg_ws)) return fail(PAD_ERR_INVALID_ARG, "tensors must be 16-byte aligned");
  const size_t need = attn_aggregate_ws_floats(n_tokens, n_segments, d_model) * sizeof(float);
  if (n_events > 0 && seg_ws_bytes < need)
    return fail(PAD_ERR_WORKSPACE_TOO_SMALL, "seg_ws has %zu bytes, the call needs %zu", seg_ws_bytes, need);
  cudaError_t e = launch_attn_aggregate(x, n_tokens, d_model, attn, offsets, n_segments, interval, n_events, g_emb,
                                        seg_ws, out, reinterpret_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? PAD_OK : cuda_fail(e, "attention aggregate launch");
}

// ---------------------------------------------------------------------------
// Full-sequence prefill / training forward (Sec. 3.4, Fig. 3)
// ---------------------------------------------------------------------------

static std::atomic<uint64_t> g_prefill_gen{0};  // generation of the last tensor-core prefill launch

pad_status pad_prefill_attn(const pad_problem* prob, int32_t prefix_len, int32_t n_branches,
                            const int32_t* branch_len, const void* q, const void* k, const void* v, void* out,
                            float* lse, pad_stream_t stream) {
  pad_status st = check_problem(prob);
  if (st != PAD_OK) return st;
  if (prefix_len < 0) return fail(PAD_ERR_INVALID_ARG, "prefix_len < 0");
  if (n_branches < 0 || n_branches > 1024) return fail(PAD_ERR_UNSUPPORTED, "n_branches=%d outside [0, 1024]", n_branches);
  if (n_branches > 0 && !branch_len) return fail(PAD_ERR_INVALID_ARG, "branch_len is NULL");
  int64_t n = prefix_len;
  for (int b = 0; b < n_branches; ++b) {
    if (branch_len[b] < 0) return fail(PAD_ERR_INVALID_ARG, "branch_len[%d]=%d < 0", b, branch_len[b]);
    n += branch_len[b];
  }
  if (n > INT32_MAX / 2) return fail(PAD_ERR_UNSUPPORTED, "sequence too long");
  if (n == 0) return PAD_OK;
  if (!q || !k || !v || !out) return fail(PAD_ERR_INVALID_ARG, "NULL tensor");
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(out) || (lse && (reinterpret_cast<uintptr_t>(lse) & 3u)))
    return fail(PAD_ERR_INVALID_ARG, "tensors must be 16-byte aligned (lse 4-byte)");
  cudaError_t e;
  if (prob->head_dim == 128 && !(prob->flags & (PAD_FLAG_PREFIX_MMA | PAD_FLAG_PREFIX_SIMT))) {
    const uint64_t gen = next_generation();
    g_prefill_gen.store(gen);
    e = launch_prefill_tc((int32_t)n, prefix_len, n_branches, branch_len, prob->h_q, prob->h_kv, prob->scale,
                          prob->out_dtype == 1, gen, q, k, v, out, lse, reinterpret_cast<cudaStream_t>(stream));
  } else {
    e = launch_prefill((int32_t)n, prefix_len, n_branches, branch_len, prob->h_q, prob->h_kv, prob->head_dim,
                       prob->scale, prob->out_dtype == 1, q, k, v, out, lse, reinterpret_cast<cudaStream_t>(stream));
  }
  return e == cudaSuccess ? PAD_OK : cuda_fail(e, "prefill launch");
}

pad_status pad_prefill_status(pad_stream_t stream) {
  PadDevHeader* hdr = nullptr;
  cudaError_t e = prefill_header(&hdr);
  if (e != cudaSuccess) return cuda_fail(e, "prefill status word");
  PadDevHeader h;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  e = cudaMemcpyAsync(&h, hdr, sizeof(h), cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(e, "reading prefill status");
  const int code = (int)(h.word & 0xffull);
  if ((h.word >> 8) == g_prefill_gen.load() && code != PAD_OK)
    return fail((pad_status)code, "prefill kernel reported %s (detail %d %d %d)", pad_status_string((pad_status)code),
                h.info[0], h.info[1], h.info[2]);
  return PAD_OK;
}
