/*
 * libpad — event-factorized parallel decode attention on GB300 (sm_103a).
 *
 * One decode step of one attention layer under the event-factorized
 * dependency structure of Sec. 3.4 (Eq. 3 and the restructured causal mask of
 * Fig. 3): every active event branch contributes one query token; the query of
 * branch e attends to the shared prefix of its video (the multimodal prefix P
 * followed by the planning tokens G^1..G^K, S of Sec. 3.3) and to its own
 * branch's private tokens (anchor, L^e_<j and the token appended at this
 * step), never to another branch's tokens.
 *
 * A step is three calls, all stream-ordered and asynchronous:
 *   pad_plan              host: validate, allocate pages, build the work list in a
 *                         library-owned page-locked image that the kernels read in
 *                         place (nothing is put on the stream);
 *   pad_kv_append         device: write each branch's new K/V into its page;
 *   pad_event_decode_attn device: shared-prefix split-KV pass, private-suffix
 *                         pass and log-sum-exp merge; writes O and LSE.
 *
 * Ownership: the caller owns every device buffer (prefix KV, page pools, page
 * table, Q, outputs, workspace); the library never allocates device memory.
 * A pad_plan_t holds host metadata and a page-locked, device-mapped image of the
 * step's descriptors (from a per-device pool of library-owned buffers, kept until
 * exit); it stays valid until pad_plan_destroy, which may follow its launches at
 * once: an image is rewritten only after the launches that read it have completed.
 * A plan is tied to the workspace it was built on, which holds the status word, the
 * split-KV partial states and the counters by which prefix CTAs tell the fused merge
 * that their partials are written; steps that share a workspace run in stream order.
 * Zero-fill a workspace once when it is allocated; every launch leaves its counters at
 * zero again, and pad_device_status zeroes them after a device error.
 *
 * Errors: every call validates its arguments on the host and returns a
 * pad_status before launching anything; pad_last_error() gives a message
 * (thread-local).  Errors found by a kernel (a page id outside the pool) set a
 * status word in the workspace, tagged with the plan's generation (a number drawn
 * per plan), which pad_device_status() reads; an error recorded by another plan's
 * kernels does not show up as this plan's.
 *
 * Layouts (row-major, element type bf16 unless stated):
 *   q          [n_events, h_q, head_dim]
 *   k_prefix   [T_total, h_kv, head_dim]   (video b's prefix starts at token
 *   v_prefix   [T_total, h_kv, head_dim]    prefix_offset[b] and has prefix_len[b] tokens)
 *   k_pool     [n_pages, h_kv, page_size, head_dim]
 *   v_pool     [n_pages, h_kv, page_size, head_dim]
 *   k_new      [n_events, h_kv, head_dim]
 *   v_new      [n_events, h_kv, head_dim]
 *   page_table [n_events, max_pages] int32 (row e belongs to event e of this step)
 *   out        [n_events, h_q, head_dim]   fp32 (out_dtype 0) or bf16 (out_dtype 1)
 *   lse        [n_events, h_q] fp32, natural log
 * q-head j reads kv-head floor(j / G) with G = h_q / h_kv.
 */
#ifndef PAD_H
#define PAD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* A CUDA stream handle (the same object as cudaStream_t); NULL = legacy default stream. */
typedef struct CUstream_st* pad_stream_t;

typedef enum {
  PAD_OK = 0,
  PAD_ERR_INVALID_ARG = 1,         /* a pointer, size, layout or length is not acceptable */
  PAD_ERR_UNSUPPORTED = 2,         /* a valid shape this build does not implement */
  PAD_ERR_OUT_OF_PAGES = 3,        /* the free pages do not cover this step's new pages */
  PAD_ERR_WORKSPACE_TOO_SMALL = 4, /* workspace_bytes < pad_workspace_size(...) */
  PAD_ERR_CUDA = 5,                /* a CUDA runtime call failed (message has the reason) */
  PAD_ERR_DEVICE_TIMEOUT = 6,      /* a bounded device-side wait gave up */
  PAD_ERR_DEVICE_BOUNDS = 7        /* a kernel met a page id outside the pool and skipped it */
} pad_status;

/* Shape of one attention layer.
 *   h_q, h_kv   query and key/value heads, h_q % h_kv == 0, G = h_q / h_kv in [1, 16]
 *   head_dim    64 or 128
 *   page_size   tokens per page of the private KV pool: 4, 8, 16, 32 or 64
 *   scale       softmax scale applied to q.k (1/sqrt(head_dim) in the paper's model)
 *   out_dtype   0 = fp32 output, 1 = bf16 output
 *   num_sms     SM count used to size the split-KV grid; 0 = query the current device
 *   flags       PAD_FLAG_* below; 0 = automatic choice of the prefix kernel */
typedef struct {
  int32_t h_q;
  int32_t h_kv;
  int32_t head_dim;
  int32_t page_size;
  float scale;
  int32_t out_dtype;
  int32_t num_sms;
  int32_t flags;
} pad_problem;

/* Force one implementation of the shared-prefix pass (tests and benchmarks). */
#define PAD_FLAG_PREFIX_SIMT 0x1   /* CUDA-core path */
#define PAD_FLAG_PREFIX_MMA 0x2    /* warp-level mma.sync path */
#define PAD_FLAG_PREFIX_TC 0x4     /* tcgen05 / TMEM / TMA path, one 128-row group per CTA */
/* tcgen05 / TMEM / TMA path with two softmax groups per CTA that take turns with the tensor
 * pipe: up to 256 query rows share each K/V tile (rows > 128), or two tile parities of the
 * same <= 128 rows alternate.  Forced only: it halves the traffic per row but doubles the
 * split partials the merge reads, and was measured no faster than PAD_FLAG_PREFIX_TC. */
#define PAD_FLAG_PREFIX_DUAL 0x10
/* Run a4 + a5 inside the tensor-core prefix kernel, after each CTA's split, where every
 * (event, kv-head) pair can take a prefix CTA and the prefix grid fits one CTA per SM
 * (pad_plan_info.fused_tail says whether it was chosen).  Off by default: the separate
 * branch/merge kernel, which starts its branch pass as prefix CTAs retire, was measured
 * faster on GB300. */
#define PAD_FLAG_FUSED_MERGE 0x8

/* ---------------------------------------------------------------------------
 * Page pool bookkeeping (host).  Tracks which pages of the private KV pool are
 * in use.  The new token of a branch whose pre-step length is a multiple of
 * page_size starts a page: pad_plan gives it the lowest-numbered free page,
 * walking events in ascending order (one new token per branch per step, Eq. 3;
 * a branch that emitted EOS simply leaves the event list, Sec. 3.4).
 * ------------------------------------------------------------------------- */
typedef struct pad_cache_state pad_cache_state;

/* Create a pool of n_pages (>= 0) pages, all free.  *out receives the handle. */
pad_status pad_cache_state_create(int32_t n_pages, pad_cache_state** out);
void pad_cache_state_destroy(pad_cache_state* cache);
/* Mark pages [n] as in use (a cache built before the library took over).
 * Fails with PAD_ERR_INVALID_ARG, changing nothing, if a page is out of range or already used. */
pad_status pad_cache_state_mark_used(pad_cache_state* cache, const int32_t* pages, int32_t n);
/* Return pages [n] to the free set (pages of branches that terminated).
 * Fails with PAD_ERR_INVALID_ARG, changing nothing, if a page is out of range or already free. */
pad_status pad_cache_state_release(pad_cache_state* cache, const int32_t* pages, int32_t n);
int32_t pad_cache_state_num_pages(const pad_cache_state* cache);
int32_t pad_cache_state_free_count(const pad_cache_state* cache);
/* Checkpoint: used[p] = 1 if page p is in use, else 0; used has num_pages entries (host). */
pad_status pad_cache_state_export(const pad_cache_state* cache, uint8_t* used);
/* Restore a checkpoint written by pad_cache_state_export (n_pages entries, host). */
pad_status pad_cache_state_import(pad_cache_state* cache, const uint8_t* used, int32_t n_pages);

/* ---------------------------------------------------------------------------
 * Planning (a1 of the step; the paper gives no kernel, so the work split is
 * this library's design: split-KV over each video's shared prefix).
 * ------------------------------------------------------------------------- */
typedef struct pad_plan_t pad_plan_t;

/* Bytes of device workspace pad_plan needs for this batch (host arrays, same
 * meaning as in pad_plan).  Returns 0 on invalid arguments. */
size_t pad_workspace_size(const pad_problem* prob, int32_t n_videos, const int32_t* prefix_len,
                          int32_t n_events, const int32_t* event_video);

/* Plan one decode step.
 *   prob           layer shape (see pad_problem)
 *   cache          page bookkeeping; pages for this step's new page starts are taken from it
 *   n_videos       videos in the batch (>= 0)
 *   prefix_len     [n_videos] host: shared-prefix tokens of each video (>= 0)
 *   prefix_offset  [n_videos] host: first token of each prefix in k_prefix/v_prefix,
 *                  or NULL for packed prefixes (exclusive prefix sum of prefix_len)
 *   n_events       active event branches this step (>= 0); 0 gives a plan that launches nothing
 *   event_video    [n_events] host: video of each event, non-decreasing, in [0, n_videos)
 *   event_len      [n_events] host: private tokens of each branch BEFORE this step's append
 *                  (at most 65534);
 *                  branch e attends to event_len[e] + 1 private keys after the append
 *   page_table     [n_events * max_pages] device: row e lists branch e's pages; the
 *                  new-page entries are written by pad_kv_append (or pad_decode_step)
 *   max_pages      columns of page_table; event_len[e] / page_size must be < max_pages
 *   workspace      device, 256-byte aligned, at least pad_workspace_size(...) bytes,
 *                  zero-filled when allocated (see above); NULL plans on the host only
 *                  (no image; the plan cannot be launched)
 *   stream         unused (kept for the interface): pad_plan enqueues nothing; it may
 *                  wait for the launches of an earlier plan whose image it reuses, once
 *                  eight or more images of the device have been released
 *   plan_out       receives the new plan (free with pad_plan_destroy)
 * On any error nothing changes: no page is taken. */
pad_status pad_plan(const pad_problem* prob, pad_cache_state* cache, int32_t n_videos,
                    const int32_t* prefix_len, const int64_t* prefix_offset, int32_t n_events,
                    const int32_t* event_video, const int32_t* event_len, int32_t* page_table,
                    int32_t max_pages, void* workspace, size_t workspace_bytes,
                    pad_stream_t stream, pad_plan_t** plan_out);

/* Page given to each event this step: new_page[e] = page id, or -1 if branch e
 * keeps writing into its current page.  new_page has n_events entries (host). */
pad_status pad_plan_new_pages(const pad_plan_t* plan, int32_t* new_page);

/* Give the pages this plan took back to `cache` (host bookkeeping only; the device page
 * table keeps its entries).  For a step that is re-run with the same lengths, such as a
 * timing loop, or a step that is abandoned.  PAD_ERR_INVALID_ARG if a page is not in use. */
pad_status pad_plan_release_new_pages(const pad_plan_t* plan, pad_cache_state* cache);

/* Rotary embedding fused into the step (host; before the plan's launches).  Sec. 3.4 gives
 * the tokens that different branches generate at the same decoding step the same position
 * index; positions[e] is the position of event e's token at this step (the caller passes
 * that shared value), and the step's kernels rotate q (every head of event e) and k_new[e]
 * at it where they load them, instead of a separate rotation pass.  V is not rotated; the
 * prefix and earlier branch keys are expected rotated already (they were, when written).
 * Rotate-half form over the whole head dimension:
 *   x'_i = x_i cos_i - x_{i+D/2} sin_i,   x'_{i+D/2} = x_{i+D/2} cos_i + x_i sin_i,
 * each product and sum rounded to fp32 and the result to bf16 (the rotated key is what the
 * pool receives), exactly as an unfused pass computing in fp32 would store it.
 *   positions  [n_events] host, each in [0, max_position)
 *   cos_sin    [max_position, head_dim] device fp32, 16-byte aligned: cos_i in columns
 *              i < D/2, sin_i in columns D/2 + i (the model's own table; read, not owned)
 * PAD_ERR_INVALID_ARG (nothing changes) for a NULL or misaligned table, or a position out
 * of range.  Applies to pad_decode_step, pad_kv_append + pad_event_decode_attn and the
 * static variant alike. */
pad_status pad_plan_set_rope(pad_plan_t* plan, const int32_t* positions, const float* cos_sin,
                             int32_t max_position);

/* Which planning tokens a branch sees (host; before the plan's launches).  The prefix of a
 * video ends with its planning tokens G^1..G^K and the end-of-planning token S (Sec. 3.3).
 *   PAD_G_ALL  (default) every branch sees all of them: the method's mask (Sec. 3.4).
 *   PAD_G_SELF the "self G-token only" structure of the paper's attention ablation
 *              (Tab. 8): event e sees P, S and G^(g_index[e]+1) only, besides its branch.
 *   n_planning [n_videos] host: K of each video (0 = nothing hidden in that video);
 *              K + 1 <= prefix_len
 *   g_index    [n_events] host: each event's own planning token, in [0, K)
 * Ignored (may be NULL) for PAD_G_ALL.  PAD_ERR_INVALID_ARG (nothing changes) on a bad
 * mode, count or index. */
#define PAD_G_ALL 0
#define PAD_G_SELF 1
pad_status pad_plan_set_g_visibility(pad_plan_t* plan, int32_t mode, const int32_t* n_planning,
                                     const int32_t* g_index);

/* Which branch tokens a branch sees (host; before the plan's launches).
 *   PAD_BRANCH_OWN    (default) only its own: the method's mask (Sec. 3.4).
 *   PAD_BRANCH_CAUSAL the "causal attention" row of the paper's attention ablation
 *                     (Tab. 8): the tokens every branch of the video generated at earlier
 *                     steps are visible to all its branches; the token a branch emits at
 *                     this step only to itself (the branches emit them simultaneously).
 * Each branch task then reads every stored branch token of its video (no sharing across
 * tasks; this variant exists for the ablation, not for speed).  PAD_ERR_INVALID_ARG on a
 * bad mode. */
#define PAD_BRANCH_OWN 0
#define PAD_BRANCH_CAUSAL 1
pad_status pad_plan_set_branch_visibility(pad_plan_t* plan, int32_t mode);

/* Summary of a plan (host): the split-KV decomposition chosen for the prefix pass. */
typedef struct {
  int32_t n_videos;
  int32_t n_events;
  int32_t n_work_items;     /* (video, kv-head, split) items of the prefix pass */
  int32_t split_len;        /* prefix tokens of the longest split (each video has its own split
                               length; a video's last split may be shorter) */
  int32_t prefix_kernel;    /* PAD_FLAG_PREFIX_* of the implementation that will run */
  int32_t n_new_pages;
  int64_t partial_rows;     /* rows of (m, l, O) partial softmax states in the workspace */
  int64_t workspace_bytes;  /* bytes of workspace this plan uses */
  int32_t param_descriptor_bytes; /* bytes of descriptors carried in each launch's parameters;
                                     0 = the kernels read them from the plan's page-locked image */
  int32_t fused_tail;       /* 1: the branch pass and the merge run inside the prefix kernel */
  uint64_t generation;      /* the number tagging this plan's device status word and counters */
  int32_t prefix_ctas;      /* CTAs of the prefix pass (a batch of videos may take several waves) */
  int32_t max_split_tiles;  /* 128-token tiles of the longest split */
  int32_t merge_first;      /* 1: in a one-call step the branch tasks wait for the prefix pass
                               before their branch pass (too few SMs are left beside it for
                               them to run there), staging the split partials meanwhile */
} pad_plan_info;
pad_status pad_plan_get_info(const pad_plan_t* plan, pad_plan_info* info);
pad_status pad_plan_destroy(pad_plan_t* plan);

/* ---------------------------------------------------------------------------
 * Device work.
 * ------------------------------------------------------------------------- */

/* a2: write k_new[e] / v_new[e] (bf16 [n_events, h_kv, head_dim], 16-byte aligned) into
 * slot event_len[e] of branch e (page page_table[e][event_len[e] / page_size], offset
 * event_len[e] % page_size) of k_pool / v_pool, and write the new page-table entries.
 * One new token per branch per step (Eq. 3).  A plan built without a workspace (host-only)
 * is accepted too: its descriptors and status word then live in the library's static scratch
 * array (see pad_event_decode_attn_static, whose rules apply), so a caller with no device
 * scratch can run a whole step as pad_kv_append + pad_event_decode_attn_static. */
pad_status pad_kv_append(const pad_plan_t* plan, const void* k_new, const void* v_new,
                         void* k_pool, void* v_pool, pad_stream_t stream);

/* a3-a5: decode attention of every active branch's query under the event-factorized
 * mask (Sec. 3.4): the shared prefix of its video plus its own event_len[e] + 1 private
 * keys (read through page_table, so pad_kv_append must precede this call on the stream).
 * All pointers device, 16-byte aligned; lse may be NULL. */
pad_status pad_event_decode_attn(const pad_plan_t* plan, const void* q, const void* k_prefix,
                                 const void* v_prefix, const void* k_pool, const void* v_pool,
                                 void* out, float* lse, pad_stream_t stream);

/* a2-a5 in one call: the same result as pad_kv_append followed by pad_event_decode_attn
 * (pools, page table, out and lse all end up identical), with one kernel launch fewer.
 * The shared-prefix pass starts the step; each (event, kv-head) branch task reads its
 * newest key from k_new / v_new, writes it into the pools (and the page table) itself,
 * and attends to it.  Arguments as in those two calls; k_pool and v_pool are written.
 * The step's first kernel uses programmatic dependent launch: it may start while the grid
 * before it on the stream is still running, if that grid releases its dependents early
 * (griddepcontrol.launch_dependents; the library's own kernels do), and it reads the first
 * tile of k_prefix / v_prefix before it waits for that grid.  Everything else it reads only
 * after that grid has completed.  So k_prefix and v_prefix must not be written by a grid
 * that releases its dependents before those writes. */
pad_status pad_decode_step(const pad_plan_t* plan, const void* q, const void* k_new, const void* v_new,
                           const void* k_prefix, const void* v_prefix, void* k_pool, void* v_pool,
                           void* out, float* lse, pad_stream_t stream);

/* ---------------------------------------------------------------------------
 * Step executor (host runtime of a serving loop; the paper has no counterpart).  It holds
 * every argument of a decode step, so that a step costs one call: pad_step_run plans the
 * step from the caller's host arrays as they are at that moment and launches it;
 * pad_step_run_host also copies this step's q, k_new and v_new in from host memory and out
 * and lse back, then waits for the stream.
 *   arguments  as pad_plan and pad_decode_step; the host arrays prefix_len, prefix_offset,
 *              event_video and event_len are borrowed (the caller keeps them alive and may
 *              change them between runs: a generation loop advances event_len in place);
 *              workspace and page_table are required
 *   options    PAD_STEP_TWO_CALL: pad_kv_append + pad_event_decode_attn instead of
 *              pad_decode_step; PAD_STEP_RELEASE_PAGES: hand the pages a run took back to
 *              the cache after launching it (to repeat one identical step, e.g. for timing);
 *              PAD_STEP_MAPPED_HOST_IO: see pad_step_run_host
 *   new_page   [n_events] host, may be NULL: the pages the run took (pad_plan_new_pages)
 * A run that fails before a kernel wrote its new pages into the page table hands them back
 * to the cache and returns the failing call's status.
 * The mask variants and RoPE are set once (pad_step_set_*: the same arguments as the
 * pad_plan_set_* calls, borrowed the same way) and apply to every later run. */
typedef struct pad_step_t pad_step_t;
#define PAD_STEP_TWO_CALL 0x1
#define PAD_STEP_RELEASE_PAGES 0x2
#define PAD_STEP_MAPPED_HOST_IO 0x4
pad_status pad_step_create(const pad_problem* prob, pad_cache_state* cache, int32_t n_videos,
                           const int32_t* prefix_len, const int64_t* prefix_offset, int32_t n_events,
                           const int32_t* event_video, const int32_t* event_len, int32_t* page_table,
                           int32_t max_pages, void* workspace, size_t workspace_bytes, const void* q,
                           const void* k_new, const void* v_new, const void* k_prefix, const void* v_prefix,
                           void* k_pool, void* v_pool, void* out, float* lse, pad_stream_t stream,
                           int32_t options, pad_step_t** step_out);
pad_status pad_step_set_rope(pad_step_t* step, const int32_t* positions, const float* cos_sin, int32_t max_position);
pad_status pad_step_set_g_visibility(pad_step_t* step, int32_t mode, const int32_t* n_planning,
                                     const int32_t* g_index);
pad_status pad_step_set_branch_visibility(pad_step_t* step, int32_t mode);
pad_status pad_step_run(pad_step_t* step, int32_t* new_page);
/*   h_q [n_events, h_q, head_dim] bf16, h_k_new / h_v_new [n_events, h_kv, head_dim] bf16,
 *   h_out [n_events, h_q, head_dim] (the problem's out_dtype), h_lse [n_events, h_q] fp32
 *   or NULL; host memory (page-locked for asynchronous copies).  The call returns after the
 *   stream has finished with them, also when it fails.  Where q, k_new and v_new
 *   follow one another in device memory and their host buffers do too, they go in one copy;
 *   so do out and lse.
 *   With PAD_STEP_MAPPED_HOST_IO, and where every host buffer is page-locked, mapped into
 *   the device's address space (cudaHostAlloc / cudaHostRegister; under unified addressing
 *   every page-locked allocation is), 16-byte aligned and lies in one such allocation (the
 *   caller's guarantee; the call checks the first and last byte), no copy engine is used:
 *   a kernel reads q, k_new and v_new over the host link into the step's device buffers, and
 *   the step's kernels write O and LSE straight into h_out and h_lse (the step's device out
 *   and lse are not written).  A buffer that fails the check sends that call down the
 *   copy path. */
pad_status pad_step_run_host(pad_step_t* step, const void* h_q, const void* h_k_new, const void* h_v_new,
                             void* h_out, float* h_lse, int32_t* new_page);
/* pad_step_enqueue_host: pad_step_run_host without the wait.  It returns once the run is on
 * the stream; the host buffers stay in use until pad_step_wait(step) returns (which waits
 * for the latest run enqueued on this step) or the stream is synchronised.  A caller with
 * several independent batches (one step executor and one set of host buffers each) plans
 * and enqueues the next batch while the device runs the previous one.  A failing enqueue
 * synchronises the stream before it returns, like pad_step_run_host. */
pad_status pad_step_enqueue_host(pad_step_t* step, const void* h_q, const void* h_k_new, const void* h_v_new,
                                 void* h_out, float* h_lse, int32_t* new_page);
pad_status pad_step_wait(pad_step_t* step);
void pad_step_destroy(pad_step_t* step);

/* Measurement aid: where a pad_step_run_host call spends its time.  After
 * pad_step_profile(step, 1) every pad_step_run_host call on the step records CUDA events on
 * the step's stream before the input copy, after it, after planning, after the launches and
 * after the output copy, reads the host clock beside each, and adds the intervals up
 * (enable 0 stops; either call clears the sums).  pad_step_profile_read writes 12 values
 * (out must hold n >= 12): out[0] the calls profiled, then means in microseconds:
 *   host    out[1] input copy call(s)   out[2] pad_plan   out[3] kernel launches
 *           out[4] output copy call(s)  out[5] stream wait  out[6] whole call
 *   device  out[7] input copy  out[8] idle until the planned launches  out[9] kernels
 *           out[10] output copy  out[11] first event to last
 * The extra event records add a little host time to each profiled call. */
pad_status pad_step_profile(pad_step_t* step, int32_t enable);
pad_status pad_step_profile_read(const pad_step_t* step, double* out, int32_t n);

/* Allocation-free variant of pad_event_decode_attn (the paper has no counterpart; this
 * is an interface for callers, not part of the method).  Same arguments and result.  It
 * is meant for callers that cannot give the library device scratch memory, for example a
 * plugin API that hands out tensors but no allocator, or a serving loop whose device
 * memory is reserved up front and must not change while it runs.  Instead of the plan's
 * workspace it uses a 16 MiB device array inside the library (held by every GPU that
 * loads the library until the process exits) for the plan image and the split-KV partial
 * states; it calls no cudaMalloc, cudaFree or other allocating routine.
 *   plan      from pad_plan; its workspace may be NULL (a host-only plan), but it must
 *             carry the page table.  Plans needing more than 16 MiB of scratch
 *             (pad_plan_get_info().workspace_bytes) fail with PAD_ERR_WORKSPACE_TOO_SMALL.
 *   The branch keys are read from the pools, so this step's K/V must already be there:
 *   call pad_kv_append with the same plan first (it also takes host-only plans).
 * The first call on a device looks up the array's device address (cudaGetSymbolAddress)
 * and caches it, so make that first call before any stream capture.  All calls share the
 * array: calls that overlap on the GPU (other streams or threads) race on it; calls in
 * order on one stream are safe (each copies the plan image into it).  That copy comes
 * from the plan's pageable host memory, so the call blocks until the driver has staged
 * it, and a graph captured around the call keeps the plan's host address: the plan must
 * outlive such a graph.  Device errors (an out-of-pool page id, a bounded wait that gave
 * up) go to the array's status word, tagged with the plan; pad_device_status(plan) reads
 * it for a plan without a workspace. */
pad_status pad_event_decode_attn_static(const pad_plan_t* plan, const void* q, const void* k_prefix,
                                        const void* v_prefix, const void* k_pool, const void* v_pool,
                                        void* out, float* lse, pad_stream_t stream);

/* ---------------------------------------------------------------------------
 * Grounding readout of the planning tokens (Sec. 3.3 and the paper's note on grounding at
 * inference by similarity matching).  Each generated event token G^i and every
 * audio-visual prefix token are first mapped by the model's projection (its two-layer
 * MLP, applied by the caller like any other layer); the dot products of G^i with the
 * tokens of one time segment are summed into a segment score, and the segments whose
 * score reaches `fraction` (0.5 or 0.7 in the paper) of the event's best score are its
 * grounded segments.  Segments are contiguous token ranges [offsets[s], offsets[s+1]).
 * Since the segment score is linear in the token features, the prefix is pooled once per
 * segment (pad_ground_pool) and every event is scored against the pooled rows
 * (pad_ground_score).  All calls are asynchronous on `stream`; argument errors return
 * before any launch.  pad_ground_pool adds partial sums of row slices with atomics: its fp32
 * results do not depend on the order beyond rounding, but are not bit-reproducible from run
 * to run.  pad_attn_aggregate sums in a fixed order: its results are the same on every run.
 * --------------------------------------------------------------------------- */

/* seg_sum[s, :] = sum of f_proj[t, :] over the tokens t of segment s (fp32).
 *   f_proj   [n_tokens, d_proj] bf16 device, 16-byte aligned; d_proj a multiple of 8, <= 2048
 *   offsets  [n_segments + 1] HOST, non-decreasing within [0, n_tokens]; 1 <= n_segments <= 1024
 *   seg_sum  [n_segments, d_proj] fp32 device, 16-byte aligned (written) */
pad_status pad_ground_pool(const void* f_proj, int64_t n_tokens, int32_t d_proj, const int32_t* offsets,
                           int32_t n_segments, float* seg_sum, pad_stream_t stream);

/* scores[i, s] = <g_proj[i], seg_sum[s]>; salient[i, s] = 1 when scores[i, s] >= fraction *
 * best_i (best_i > 0), else only the first best segment; interval[i] = (first, last)
 * salient segment.
 *   g_proj   [n_events, d_proj] bf16 device, 16-byte aligned
 *   scores   [n_events, n_segments] fp32, salient [n_events, n_segments] uint8,
 *   interval [n_events, 2] int32, all device (written); fraction in [0, 1] */
pad_status pad_ground_score(const void* g_proj, int32_t n_events, const float* seg_sum, int32_t n_segments,
                            int32_t d_proj, float fraction, float* scores, uint8_t* salient, int32_t* interval,
                            pad_stream_t stream);

/* Attention-guided aggregation (Sec. 3.3, strategy (3)): for event i, the prefix tokens of
 * its grounded segments interval[i] = (lo, hi), i.e. tokens [offsets[lo], offsets[hi + 1]),
 * are pooled with weights attn[t] (the attention of the last text-query token on them) and
 * out[i] = g_emb[i] + sum_t attn[t] x[t] / sum_t attn[t] (g_emb[i] alone when that weight is 0).
 * The weights belong to the tokens, so the hidden states are pooled once, per piece of at
 * most 256 tokens of a segment, into seg_ws (weighted row sums, then the pieces' weight
 * sums), and each event adds up the pieces of its segments; overlapping intervals read x
 * once.
 *   x        [n_tokens, d_model] bf16 device (prefix hidden states), 16-byte aligned;
 *            d_model a multiple of 8
 *   attn     [n_tokens] fp32 device; interval [n_events, 2] int32 device (as written by
 *            pad_ground_score; clamped to the segments); offsets as above (host)
 *   g_emb    [n_events, d_model] bf16 device, 16-byte aligned
 *   seg_ws   device scratch of seg_ws_bytes >= pad_attn_aggregate_workspace_size(n_tokens,
 *            n_segments, d_model) = (n_segments + ceil(n_tokens / 256)) * (d_model + 1) * 4
 *            bytes, 16-byte aligned (overwritten; owned by the caller, free for reuse once
 *            the call's work on `stream` is done); too small: PAD_ERR_WORKSPACE_TOO_SMALL
 *   out      [n_events, d_model] fp32 device (written) */
size_t pad_attn_aggregate_workspace_size(int64_t n_tokens, int32_t n_segments, int32_t d_model);
pad_status pad_attn_aggregate(const void* x, int64_t n_tokens, int32_t d_model, const float* attn,
                              const int32_t* offsets, int32_t n_segments, const int32_t* interval, int32_t n_events,
                              const void* g_emb, float* seg_ws, size_t seg_ws_bytes, float* out,
                              pad_stream_t stream);

/* Forward attention of a whole sequence under the event-factorized mask (Sec. 3.4, Fig. 3),
 * as training with teacher forcing (and a prefill of the branches) needs it: the sequence of
 * one video is [prefix of prefix_len tokens (P, G^1..G^K, S) ; branch 0 ; ... ; branch E-1],
 * branch b holding branch_len[b] tokens (its anchor and local tokens).  A prefix token
 * attends causally within the prefix; a branch token attends to the whole prefix and
 * causally to its own branch; never to another branch.  Block-sparse: each query tile reads
 * only the key ranges its rows can see.
 *   prob        h_q, h_kv, head_dim (64 or 128), scale, out_dtype (num_sms, flags, page_size
 *               unused)
 *   branch_len  [n_branches] HOST, each >= 0; n_branches <= 1024
 *   q           [N, h_q, head_dim] bf16, k / v [N, h_kv, head_dim] bf16, N = prefix_len +
 *               sum(branch_len), token-major; out [N, h_q, head_dim] fp32 or bf16; lse [N, h_q]
 *               fp32 (natural log) or NULL; all device, 16-byte aligned (lse 4-byte)
 * One video per call; the work is asynchronous on `stream`.  head_dim 128 runs on the
 * tensor-core kernel (a CTA: 128 / G tokens x the G heads of one kv-head against its visible
 * key ranges, output normalised in place); head_dim 64, or flags PAD_FLAG_PREFIX_MMA, on the
 * warp-level kernel (64 tokens x one head). */
pad_status pad_prefill_attn(const pad_problem* prob, int32_t prefix_len, int32_t n_branches,
                            const int32_t* branch_len, const void* q, const void* k, const void* v, void* out,
                            float* lse, pad_stream_t stream);

/* Synchronise the stream and read the status word of the last tensor-core prefill launch
 * (a bounded wait that gave up: PAD_ERR_DEVICE_TIMEOUT); PAD_OK otherwise. */
pad_status pad_prefill_status(pad_stream_t stream);

/* Synchronise the stream and read the plan's device status word:
 * PAD_OK, PAD_ERR_DEVICE_BOUNDS or PAD_ERR_DEVICE_TIMEOUT.  For a plan without a workspace
 * the word is the static scratch array's (pad_event_decode_attn_static); PAD_OK if no call
 * has used that array on the current device. */
pad_status pad_device_status(const pad_plan_t* plan, pad_stream_t stream);

/* Message for the last error on this thread ("" if none). */
const char* pad_last_error(void);
const char* pad_status_string(pad_status status);

/* ---------------------------------------------------------------------------
 * Measurement aid: CUDA-event timing of the dominant kernel (the shared-prefix
 * pass).  After pad_timing_enable(n), the next n pad_event_decode_attn calls
 * record an event pair around that kernel on the call's stream;
 * pad_timing_read synchronises those events and returns the summed time in ms
 * and the number of launches timed, then disables timing.  Process-global; not
 * for concurrent use from several threads.
 * ------------------------------------------------------------------------- */
pad_status pad_timing_enable(int32_t max_launches);
pad_status pad_timing_read(float* total_ms, int32_t* n_launches);

#ifdef __cplusplus
}
#endif

#endif /* PAD_H */
