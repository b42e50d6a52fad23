"""ctypes binding of libpad (include/pad.h): argument marshalling only.

Every step of the decode path runs in the CUDA library; this module converts
torch tensors to device pointers, numpy arrays to host pointers, and status
codes to exceptions.  It fails loudly when libpad.so has not been built.
"""
from __future__ import annotations

import ctypes
import os
from ctypes import POINTER, c_float, c_int32, c_int64, c_size_t, c_uint8, c_void_p

import numpy as np

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libpad.so")
_lib = None

PAD_OK = 0
STATUS_NAMES = {
    0: "PAD_OK", 1: "PAD_ERR_INVALID_ARG", 2: "PAD_ERR_UNSUPPORTED", 3: "PAD_ERR_OUT_OF_PAGES",
    4: "PAD_ERR_WORKSPACE_TOO_SMALL", 5: "PAD_ERR_CUDA", 6: "PAD_ERR_DEVICE_TIMEOUT",
    7: "PAD_ERR_DEVICE_BOUNDS",
}
FLAG_PREFIX_SIMT = 0x1
FLAG_PREFIX_MMA = 0x2
FLAG_PREFIX_TC = 0x4
FLAG_FUSED_MERGE = 0x8
FLAG_PREFIX_DUAL = 0x10
G_ALL = 0
G_SELF = 1
BRANCH_OWN = 0
BRANCH_CAUSAL = 1


class PadError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {message}")
        self.status = status


class Problem(ctypes.Structure):
    _fields_ = [("h_q", c_int32), ("h_kv", c_int32), ("head_dim", c_int32),
                ("page_size", c_int32), ("scale", c_float), ("out_dtype", c_int32),
                ("num_sms", c_int32), ("flags", c_int32)]


class PlanInfo(ctypes.Structure):
    _fields_ = [("n_videos", c_int32), ("n_events", c_int32), ("n_work_items", c_int32),
                ("split_len", c_int32), ("prefix_kernel", c_int32), ("n_new_pages", c_int32),
                ("partial_rows", c_int64), ("workspace_bytes", c_int64),
                ("param_descriptor_bytes", c_int32), ("fused_tail", c_int32),
                ("generation", ctypes.c_uint64), ("prefix_ctas", c_int32), ("max_split_tiles", c_int32),
                ("merge_first", c_int32)]


_I32P = POINTER(c_int32)
_I64P = POINTER(c_int64)

# name -> (restype, argtypes); mirrors include/pad.h
_SIGNATURES = {
    "pad_cache_state_create": (c_int32, [c_int32, POINTER(c_void_p)]),
    "pad_cache_state_destroy": (None, [c_void_p]),
    "pad_cache_state_mark_used": (c_int32, [c_void_p, _I32P, c_int32]),
    "pad_cache_state_release": (c_int32, [c_void_p, _I32P, c_int32]),
    "pad_cache_state_num_pages": (c_int32, [c_void_p]),
    "pad_cache_state_free_count": (c_int32, [c_void_p]),
    "pad_cache_state_export": (c_int32, [c_void_p, POINTER(c_uint8)]),
    "pad_cache_state_import": (c_int32, [c_void_p, POINTER(c_uint8), c_int32]),
    "pad_workspace_size": (c_size_t, [POINTER(Problem), c_int32, _I32P, c_int32, _I32P]),
    "pad_plan": (c_int32, [POINTER(Problem), c_void_p, c_int32, _I32P, _I64P, c_int32, _I32P,
                           _I32P, c_void_p, c_int32, c_void_p, c_size_t, c_void_p,
                           POINTER(c_void_p)]),
    "pad_plan_new_pages": (c_int32, [c_void_p, _I32P]),
    "pad_plan_release_new_pages": (c_int32, [c_void_p, c_void_p]),
    "pad_step_create": (c_int32, [POINTER(Problem), c_void_p, c_int32, _I32P, _I64P, c_int32, _I32P, _I32P,
                                  c_void_p, c_int32, c_void_p, c_size_t] + [c_void_p] * 10
                        + [c_int32, POINTER(c_void_p)]),
    "pad_step_set_rope": (c_int32, [c_void_p, _I32P, c_void_p, c_int32]),
    "pad_step_set_g_visibility": (c_int32, [c_void_p, c_int32, _I32P, _I32P]),
    "pad_step_set_branch_visibility": (c_int32, [c_void_p, c_int32]),
    "pad_step_run": (c_int32, [c_void_p, _I32P]),
    "pad_step_run_host": (c_int32, [c_void_p] * 6 + [_I32P]),
    "pad_step_destroy": (None, [c_void_p]),
    "pad_plan_set_rope": (c_int32, [c_void_p, _I32P, c_void_p, c_int32]),
    "pad_plan_set_g_visibility": (c_int32, [c_void_p, c_int32, _I32P, _I32P]),
    "pad_plan_set_branch_visibility": (c_int32, [c_void_p, c_int32]),
    "pad_plan_get_info": (c_int32, [c_void_p, POINTER(PlanInfo)]),
    "pad_plan_destroy": (c_int32, [c_void_p]),
    "pad_kv_append": (c_int32, [c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p]),
    "pad_event_decode_attn": (c_int32, [c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                                        c_void_p, c_void_p, c_void_p, c_void_p]),
    "pad_event_decode_attn_static": (c_int32, [c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                                               c_void_p, c_void_p, c_void_p, c_void_p]),
    "pad_decode_step": (c_int32, [c_void_p] * 11),
    "pad_prefill_attn": (c_int32, [POINTER(Problem), c_int32, c_int32, _I32P, c_void_p, c_void_p, c_void_p,
                                   c_void_p, c_void_p, c_void_p]),
    "pad_prefill_status": (c_int32, [c_void_p]),
    "pad_ground_pool": (c_int32, [c_void_p, c_int64, c_int32, _I32P, c_int32, c_void_p, c_void_p]),
    "pad_ground_score": (c_int32, [c_void_p, c_int32, c_void_p, c_int32, c_int32, c_float, c_void_p, c_void_p,
                                   c_void_p, c_void_p]),
    "pad_attn_aggregate": (c_int32, [c_void_p, c_int64, c_int32, c_void_p, _I32P, c_int32, c_void_p, c_int32,
                                     c_void_p, c_void_p, ctypes.c_size_t, c_void_p, c_void_p]),
    "pad_attn_aggregate_workspace_size": (ctypes.c_size_t, [c_int64, c_int32, c_int32]),
    "pad_device_status": (c_int32, [c_void_p, c_void_p]),
    "pad_last_error": (ctypes.c_char_p, []),
    "pad_status_string": (ctypes.c_char_p, [c_int32]),
    "pad_step_enqueue_host": (c_int32, [c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, _I32P]),
    "pad_step_wait": (c_int32, [c_void_p]),
    "pad_step_profile": (c_int32, [c_void_p, c_int32]),
    "pad_step_profile_read": (c_int32, [c_void_p, POINTER(ctypes.c_double), c_int32]),
    "pad_timing_enable": (c_int32, [c_int32]),
    "pad_timing_read": (c_int32, [POINTER(c_float), _I32P]),
}


def lib_path() -> str:
    return _LIB_PATH


def lib():
    """Load libpad.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(_LIB_PATH):
            raise RuntimeError(f"libpad.so is not built ({_LIB_PATH}); run "
                               "`python -c 'import __graft_entry__ as g; g.build()'`")
        L = ctypes.CDLL(_LIB_PATH)
        for name, (res, args) in _SIGNATURES.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


def _check(status: int):
    if status != PAD_OK:
        msg = lib().pad_last_error().decode(errors="replace")
        raise PadError(status, msg)


def _i32(a):
    a = np.ascontiguousarray(a, dtype=np.int32)
    return a, a.ctypes.data_as(_I32P)


def _ptr(t):
    """Device pointer of a tensor (None -> NULL)."""
    if t is None:
        return None
    if not t.is_contiguous():
        raise ValueError("tensors passed to libpad must be contiguous")
    return c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        import torch
        return c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, int):
        return c_void_p(stream)
    return c_void_p(stream.cuda_stream)


def make_problem(h_q, h_kv, head_dim, page_size=16, scale=None, out_dtype=0, num_sms=0, flags=0):
    if scale is None:
        scale = 1.0 / float(head_dim) ** 0.5
    return Problem(h_q, h_kv, head_dim, page_size, scale, out_dtype, num_sms, flags)


class CacheState:
    """Host bookkeeping of the private-KV page pool (pad_cache_state)."""

    def __init__(self, n_pages: int, used_pages=None):
        h = c_void_p()
        _check(lib().pad_cache_state_create(int(n_pages), ctypes.byref(h)))
        self._h = h
        if used_pages is not None and len(used_pages):
            self.mark_used(used_pages)

    @property
    def handle(self):
        return self._h

    def mark_used(self, pages):
        a, p = _i32(pages)
        _check(lib().pad_cache_state_mark_used(self._h, p, int(a.size)))

    def release(self, pages):
        a, p = _i32(pages)
        _check(lib().pad_cache_state_release(self._h, p, int(a.size)))

    @property
    def n_pages(self) -> int:
        return int(lib().pad_cache_state_num_pages(self._h))

    @property
    def free_count(self) -> int:
        return int(lib().pad_cache_state_free_count(self._h))

    def export(self) -> np.ndarray:
        out = np.zeros(self.n_pages, dtype=np.uint8)
        _check(lib().pad_cache_state_export(self._h, out.ctypes.data_as(POINTER(c_uint8))))
        return out

    def import_(self, used: np.ndarray):
        u = np.ascontiguousarray(used, dtype=np.uint8)
        _check(lib().pad_cache_state_import(self._h, u.ctypes.data_as(POINTER(c_uint8)), int(u.size)))

    def free_pages(self) -> np.ndarray:
        return np.nonzero(self.export() == 0)[0].astype(np.int32)

    def __del__(self):
        if getattr(self, "_h", None) is not None and _lib is not None:
            _lib.pad_cache_state_destroy(self._h)
            self._h = None


class Plan:
    """A planned decode step (pad_plan_t)."""

    def __init__(self, handle, n_events):
        self._h = handle
        self.n_events = n_events

    @property
    def handle(self):
        return self._h

    def new_pages(self) -> np.ndarray:
        out = np.full(self.n_events, -1, dtype=np.int32)
        _check(lib().pad_plan_new_pages(self._h, out.ctypes.data_as(_I32P)))
        return out

    def release_new_pages(self, cache: "CacheState"):
        """Give the pages this plan took back to ``cache`` (pad_plan_release_new_pages)."""
        _check(lib().pad_plan_release_new_pages(self._h, cache.handle))

    def set_rope(self, positions, cos_sin, max_position: int = None):
        """Rotate q and k_new at these per-event positions in the step's kernels
        (pad_plan_set_rope); ``cos_sin`` is the device fp32 table [max_position, D]."""
        pos = np.ascontiguousarray(positions, dtype=np.int32)
        n = int(cos_sin.shape[0]) if max_position is None else int(max_position)
        _check(lib().pad_plan_set_rope(self._h, pos.ctypes.data_as(_I32P), _ptr(cos_sin), n))

    def set_g_visibility(self, mode: int, n_planning=None, g_index=None):
        """pad_plan_set_g_visibility: G_SELF hides the other events' planning tokens."""
        if n_planning is None or g_index is None:
            _check(lib().pad_plan_set_g_visibility(self._h, int(mode), None, None))
            return
        k = np.ascontiguousarray(n_planning, dtype=np.int32)
        g = np.ascontiguousarray(g_index, dtype=np.int32)
        _check(lib().pad_plan_set_g_visibility(self._h, mode, k.ctypes.data_as(_I32P),
                                               g.ctypes.data_as(_I32P)))

    def set_branch_visibility(self, mode: int):
        """pad_plan_set_branch_visibility: BRANCH_CAUSAL shows every branch's stored tokens."""
        _check(lib().pad_plan_set_branch_visibility(self._h, int(mode)))

    def info(self) -> dict:
        i = PlanInfo()
        _check(lib().pad_plan_get_info(self._h, ctypes.byref(i)))
        return {f: getattr(i, f) for f, _ in PlanInfo._fields_}

    def destroy(self):
        if self._h is not None and _lib is not None:
            _lib.pad_plan_destroy(self._h)
            self._h = None

    def __del__(self):
        self.destroy()


def pad_workspace_size(problem: Problem, prefix_len, event_video) -> int:
    pl, plp = _i32(prefix_len)
    ev, evp = _i32(event_video)
    return int(lib().pad_workspace_size(ctypes.byref(problem), int(pl.size), plp, int(ev.size), evp))


def pad_plan(problem: Problem, cache: CacheState, prefix_len, event_video, event_len,
             page_table=None, max_pages: int = 0, workspace=None, prefix_offset=None,
             stream=None) -> Plan:
    """Plan one decode step (host).  page_table / workspace are device tensors
    (int32 [E, max_pages] / uint8 [bytes]); workspace=None plans on the host only."""
    pl, plp = _i32(prefix_len)
    ev, evp = _i32(event_video)
    el, elp = _i32(event_len)
    po = None
    if prefix_offset is not None:
        po_arr = np.ascontiguousarray(prefix_offset, dtype=np.int64)
        po = po_arr.ctypes.data_as(_I64P)
    if page_table is not None and max_pages == 0:
        max_pages = int(page_table.shape[-1])
    ws_ptr = _ptr(workspace)
    ws_bytes = int(workspace.numel() * workspace.element_size()) if workspace is not None else 0
    strm = _stream(stream) if workspace is not None else c_void_p(0)
    h = c_void_p()
    _check(lib().pad_plan(ctypes.byref(problem), cache.handle, int(pl.size), plp, po, int(ev.size),
                          evp, elp, _ptr(page_table), int(max_pages), ws_ptr, ws_bytes, strm,
                          ctypes.byref(h)))
    return Plan(h, int(el.size))


def pad_kv_append(plan: Plan, k_new, v_new, k_pool, v_pool, stream=None):
    _check(lib().pad_kv_append(plan.handle, _ptr(k_new), _ptr(v_new), _ptr(k_pool), _ptr(v_pool),
                               _stream(stream)))


def pad_event_decode_attn(plan: Plan, q, k_prefix, v_prefix, k_pool, v_pool, out, lse=None,
                          stream=None):
    _check(lib().pad_event_decode_attn(plan.handle, _ptr(q), _ptr(k_prefix), _ptr(v_prefix),
                                       _ptr(k_pool), _ptr(v_pool), _ptr(out), _ptr(lse),
                                       _stream(stream)))


def pad_decode_step(plan: Plan, q, k_new, v_new, k_prefix, v_prefix, k_pool, v_pool, out, lse=None,
                    stream=None):
    """pad_kv_append + pad_event_decode_attn in one call (one kernel launch fewer)."""
    _check(lib().pad_decode_step(plan.handle, _ptr(q), _ptr(k_new), _ptr(v_new), _ptr(k_prefix),
                                 _ptr(v_prefix), _ptr(k_pool), _ptr(v_pool), _ptr(out), _ptr(lse),
                                 _stream(stream)))


def pad_prefill_attn(problem, prefix_len: int, branch_len, q, k, v, out, lse=None, stream=None):
    """Whole-sequence forward attention under the event-factorized mask (training / prefill)."""
    bl = np.ascontiguousarray(branch_len, dtype=np.int32)
    _check(lib().pad_prefill_attn(ctypes.byref(problem), int(prefix_len), int(bl.size), bl.ctypes.data_as(_I32P),
                                  _ptr(q), _ptr(k), _ptr(v), _ptr(out), _ptr(lse), _stream(stream)))


def pad_prefill_status(stream=None):
    """Status word of the last tensor-core prefill launch (synchronises the stream)."""
    _check(lib().pad_prefill_status(_stream(stream)))


def pad_ground_pool(f_proj, offsets, seg_sum, stream=None):
    """Per-segment sums of the projected prefix features (Sec. 3.3 grounding readout)."""
    off = np.ascontiguousarray(offsets, dtype=np.int32)
    _check(lib().pad_ground_pool(_ptr(f_proj), int(f_proj.shape[0]), int(f_proj.shape[1]),
                                 off.ctypes.data_as(_I32P), int(off.size - 1), _ptr(seg_sum), _stream(stream)))


def pad_ground_score(g_proj, seg_sum, fraction, scores, salient, interval, stream=None):
    """Segment scores, salient segments and grounded interval of every event token."""
    _check(lib().pad_ground_score(_ptr(g_proj), int(g_proj.shape[0]), _ptr(seg_sum), int(seg_sum.shape[0]),
                                  int(seg_sum.shape[1]), float(fraction), _ptr(scores), _ptr(salient),
                                  _ptr(interval), _stream(stream)))


def aggregate_workspace(n_tokens, n_segments, d_model, device="cuda"):
    """Scratch for pad_attn_aggregate (pad_attn_aggregate_workspace_size bytes of fp32)."""
    import torch
    n = int(lib().pad_attn_aggregate_workspace_size(int(n_tokens), int(n_segments), int(d_model)))
    return torch.empty(max(1, n // 4), dtype=torch.float32, device=device)


def pad_attn_aggregate(x, attn, offsets, interval, g_emb, out, seg_ws, stream=None):
    """Attention-guided pooling of each event's grounded tokens, added to its embedding
    (seg_ws: aggregate_workspace(n_tokens, n_segments, d_model))."""
    off = np.ascontiguousarray(offsets, dtype=np.int32)
    _check(lib().pad_attn_aggregate(_ptr(x), int(x.shape[0]), int(x.shape[1]), _ptr(attn),
                                    off.ctypes.data_as(_I32P), int(off.size - 1), _ptr(interval),
                                    int(g_emb.shape[0]), _ptr(g_emb), _ptr(seg_ws),
                                    int(seg_ws.numel() * seg_ws.element_size()), _ptr(out), _stream(stream)))


def pad_event_decode_attn_static(plan: Plan, q, k_prefix, v_prefix, k_pool, v_pool, out, lse=None,
                                 stream=None):
    """pad_event_decode_attn with the library's static scratch instead of a workspace."""
    _check(lib().pad_event_decode_attn_static(plan.handle, _ptr(q), _ptr(k_prefix), _ptr(v_prefix),
                                              _ptr(k_pool), _ptr(v_pool), _ptr(out), _ptr(lse),
                                              _stream(stream)))


def pad_device_status(plan: Plan, stream=None):
    _check(lib().pad_device_status(plan.handle, _stream(stream)))


def pad_timing_enable(max_launches: int):
    _check(lib().pad_timing_enable(int(max_launches)))


def pad_timing_read():
    ms = c_float()
    n = c_int32()
    _check(lib().pad_timing_read(ctypes.byref(ms), ctypes.byref(n)))
    return float(ms.value), int(n.value)


STEP_TWO_CALL = 0x1
STEP_RELEASE_PAGES = 0x2
STEP_MAPPED_HOST_IO = 0x4


class NativeStep:
    """The library's step executor (pad_step_*): every argument marshalled once in C, so a
    step is one call (``run``), or one call with the host copies and the wait included
    (``run_host``).  ``event_len`` is borrowed: update it in place between runs (a
    generation loop), the next run plans from its current values."""

    def __init__(self, problem: Problem, cache: CacheState, prefix_len, event_video, event_len,
                 page_table, max_pages, workspace, prefix_offset, q, k_new, v_new, k_prefix,
                 v_prefix, k_pool, v_pool, out, lse, stream, release_pages=True, one_call=True,
                 rope=None, self_g=None, causal=False, mapped_host_io=False):
        self.L = lib()
        self.problem = problem
        self.cache = cache
        self.prefix_len = np.ascontiguousarray(prefix_len, dtype=np.int32)
        self.event_video = np.ascontiguousarray(event_video, dtype=np.int32)
        # the executor reads this array at every run
        self.event_len = np.array(event_len, dtype=np.int32, copy=True)
        self.prefix_offset = (None if prefix_offset is None
                              else np.ascontiguousarray(prefix_offset, dtype=np.int64))
        self._keep = [q, k_new, v_new, k_prefix, v_prefix, k_pool, v_pool, out, lse, workspace, page_table]
        self.ne = int(self.event_video.size)
        opts = ((0 if one_call else STEP_TWO_CALL) | (STEP_RELEASE_PAGES if release_pages else 0)
                | (STEP_MAPPED_HOST_IO if mapped_host_io else 0))
        h = c_void_p()
        _check(self.L.pad_step_create(
            ctypes.byref(problem), cache.handle, int(self.prefix_len.size), self.prefix_len.ctypes.data_as(_I32P),
            None if self.prefix_offset is None else self.prefix_offset.ctypes.data_as(_I64P), self.ne,
            self.event_video.ctypes.data_as(_I32P), self.event_len.ctypes.data_as(_I32P), _ptr(page_table),
            int(max_pages), _ptr(workspace), int(workspace.numel() * workspace.element_size()), _ptr(q),
            _ptr(k_new), _ptr(v_new), _ptr(k_prefix), _ptr(v_prefix), _ptr(k_pool), _ptr(v_pool), _ptr(out),
            _ptr(lse), _stream(stream), opts, ctypes.byref(h)))
        self.handle = h
        if rope is not None:
            self.rope_pos = np.ascontiguousarray(rope[0], dtype=np.int32)
            self._keep.append(rope[1])
            _check(self.L.pad_step_set_rope(h, self.rope_pos.ctypes.data_as(_I32P), _ptr(rope[1]),
                                            int(rope[1].shape[0])))
        if self_g is not None:
            self.g_k = np.ascontiguousarray(self_g[0], dtype=np.int32)
            self.g_i = np.ascontiguousarray(self_g[1], dtype=np.int32)
            _check(self.L.pad_step_set_g_visibility(h, G_SELF, self.g_k.ctypes.data_as(_I32P),
                                                    self.g_i.ctypes.data_as(_I32P)))
        if causal:
            _check(self.L.pad_step_set_branch_visibility(h, BRANCH_CAUSAL))
        self.new_page = np.full(self.ne, -1, dtype=np.int32)
        self._np = self.new_page.ctypes.data_as(_I32P)
        self._run = self.L.pad_step_run
        self._run_host = self.L.pad_step_run_host

    def __call__(self):
        _check(self._run(self.handle, self._np))

    def run_host(self, h_q, h_k_new, h_v_new, h_out, h_lse=None):
        """Host tensors (page-locked): copies in, the step, copies out, stream wait (with
        mapped_host_io, the inputs are read and the outputs written by kernels over the host
        link where every buffer is page-locked and device-mapped)."""
        _check(self._run_host(self.handle, h_q.data_ptr(), h_k_new.data_ptr(), h_v_new.data_ptr(), h_out.data_ptr(),
                              None if h_lse is None else h_lse.data_ptr(), self._np))

    def enqueue_host(self, h_q, h_k_new, h_v_new, h_out, h_lse=None):
        """run_host without the wait: the buffers stay in use until wait()."""
        _check(self.L.pad_step_enqueue_host(self.handle, h_q.data_ptr(), h_k_new.data_ptr(), h_v_new.data_ptr(),
                                            h_out.data_ptr(), None if h_lse is None else h_lse.data_ptr(),
                                            self._np))

    def wait(self):
        _check(self.L.pad_step_wait(self.handle))

    PROFILE_KEYS = ("host_h2d_call", "host_plan", "host_launch", "host_d2h_call", "host_wait",
                    "host_total", "dev_h2d", "dev_idle_until_launch", "dev_kernels", "dev_d2h",
                    "dev_span")

    def profile(self, enable=True):
        """Per-phase timing of run_host (pad_step_profile); read it with profile_read."""
        _check(self.L.pad_step_profile(self.handle, 1 if enable else 0))

    def profile_read(self):
        buf = (ctypes.c_double * 12)()
        _check(self.L.pad_step_profile_read(self.handle, buf, 12))
        d = dict(zip(self.PROFILE_KEYS, list(buf)[1:]))
        d["calls"] = int(buf[0])
        return d

    def __del__(self):
        h = getattr(self, "handle", None)
        if h is not None and h.value:
            self.L.pad_step_destroy(h)
            self.handle = None
