#!/usr/bin/env python3
"""Throughput of one event-factorized parallel decode step (one attention layer) on GB300.

A step is the whole hot path: pad_plan (host work list + page allocation, carried
in the launch parameters), pad_kv_append (each branch's new K/V into its page) and
pad_event_decode_attn (shared-prefix split-KV pass, private-suffix pass and
log-sum-exp merge).  The default workload is the long-video case: batch 1,
H_q=28, H_kv=4, head_dim 128, shared prefix 32768 tokens, 32 events with private
lengths uniform in [0, 128], K with per-channel LogNormal(0, 0.5) scale.

Timing: W warm-up steps, then exactly K steps between CUDA events on the
launching stream; every step uses the next of several cold replicas of the whole
device state (their total exceeds 3x the L2 size), so each step reads from HBM.
The JSON line also carries:
  roofline      the shared-prefix kernel: algorithmic bytes (prefix K+V read once)
                per launch / its event-timed duration, against the measured HBM peak;
  e2e           the same metric through the C ABI with host buffers: H2D of the
                step's inputs (q, k_new, v_new) from pinned memory and D2H of the
                outputs (O, LSE) inside the timed region, synchronised every step;
  cpu_baseline  the fp64 oracle on this host's cores over a bounded sample;
  clocks        NVML SM clock and clock-event reasons sampled during the timed loop.

Multi-GPU: the path does not shard (one GPU, no collectives); with N ranks every
rank runs an independent replica of the step ("replicas only"), and value is
the events of all ranks divided by the slowest rank's time.

--impl reference times the fp64 oracle (the only other implementation) on the
host cores with the same metric; each step is a bounded sample of the workload.

--sweep prints one JSON line per event count E of the sweep workload (prefix 16384,
L = 48): our step's time and HBM rate, and a naive comparator that re-reads the shared
prefix once per event (one scaled_dot_product_attention call per event over that event's
own [prefix ; branch] keys, a library kernel used only as a baseline here).
"""
from __future__ import annotations

import argparse
import ctypes
import hashlib
import json
import os
import statistics
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "event-tokens/s per decode step per layer; achieved HBM GB/s vs ~8 TB/s roofline"
UNIT = "event-tokens/s"
FALLBACK_HBM_GBS = 6800.0

WORKLOADS = {
    "long_32k": "batch 1, H_q 28, H_kv 4, D 128, prefix 32768 (32736 audio-visual + 32 planning), "
                "E 32, private lengths uniform [0,128], K per-channel LogNormal(0,0.5) scale",
    "gqa_8k": "batch 1, H_q 28, H_kv 4, D 128, prefix 8192, E 8, private lengths uniform [0,64]",
    "ragged": "16 videos, H_q 28, H_kv 4, D 128, prefix uniform [4096,16384]+16, "
              "E per video uniform [4,24], private lengths uniform [0,96]",
    "tiny": "batch 1, H_q 4, H_kv 1, D 64, prefix 512, E 4, private lengths {0,5,11,16}",
}
for _E in (1, 2, 4, 8, 16, 32, 64):
    WORKLOADS[f"sweep_e{_E}"] = f"batch 1, H_q 28, H_kv 4, D 128, prefix 16384, E {_E}, private length 48"


def make_workload(name):
    from paper_2607_02963_gb300 import synth
    if name == "long_32k":
        return synth.long_32k()
    if name == "gqa_8k":
        return synth.gqa_8k()
    if name == "ragged":
        return synth.ragged_serving()
    if name == "tiny":
        return synth.tiny()
    if name.startswith("sweep_e"):
        return synth.event_sweep(int(name[len("sweep_e"):]))
    raise SystemExit(f"unknown workload {name}")


# ---------------------------------------------------------------------------
# Distributed helpers (replicas only: a barrier and max/sum reductions)
# ---------------------------------------------------------------------------

def dist_env():
    return int(os.environ.get("RANK", 0)), int(os.environ.get("WORLD_SIZE", 1)), \
        int(os.environ.get("LOCAL_RANK", 0))


def init_dist(backend):
    import torch.distributed as dist
    rank, world, _ = dist_env()
    if world > 1 and not dist.is_initialized():
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        dist.init_process_group(backend=backend, rank=rank, world_size=world)
    return rank, world


def barrier(device=None):
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized():
        if device is not None and device.type == "cuda":
            dist.barrier(device_ids=[device.index])
        else:
            dist.barrier()


def aggregate(units: float, ms: float, device=None):
    """(sum of units over ranks, max of ms over ranks)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()):
        return units, ms
    dev = device if device is not None else torch.device("cpu")
    u = torch.tensor([units], dtype=torch.float64, device=dev)
    t = torch.tensor([ms], dtype=torch.float64, device=dev)
    dist.all_reduce(u, op=dist.ReduceOp.SUM)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(u.item()), float(t.item())


# ---------------------------------------------------------------------------
# Clock sampling through NVML (read-only)
# ---------------------------------------------------------------------------

_REASONS = {0x1: "gpu_idle", 0x2: "applications_clocks_setting", 0x4: "sw_power_cap",
            0x8: "hw_slowdown", 0x10: "sync_boost", 0x20: "sw_thermal_slowdown",
            0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown",
            0x100: "display_clock_setting"}


class ClockSampler:
    def __init__(self, torch_index=0, period_s=0.005):
        self.period = period_s
        self.samples = []
        self.max_mhz = None
        self.ok = False
        self._stop = threading.Event()
        self._thread = None
        try:
            nv = ctypes.CDLL("libnvidia-ml.so.1")
            if nv.nvmlInit_v2() != 0:
                return
            h = ctypes.c_void_p()
            found = False
            try:
                import torch
                uuid = str(torch.cuda.get_device_properties(torch_index).uuid)
                if not uuid.startswith("GPU-"):
                    uuid = "GPU-" + uuid
                found = nv.nvmlDeviceGetHandleByUUID(uuid.encode(), ctypes.byref(h)) == 0
            except Exception:
                found = False
            if not found and nv.nvmlDeviceGetHandleByIndex_v2(torch_index, ctypes.byref(h)) != 0:
                return
            self.nv, self.h = nv, h
            mx = ctypes.c_uint()
            if nv.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(mx)) == 0:
                self.max_mhz = int(mx.value)
            fn = getattr(nv, "nvmlDeviceGetCurrentClocksEventReasons", None)
            self._reasons_fn = fn or getattr(nv, "nvmlDeviceGetCurrentClocksThrottleReasons")
            self.ok = True
        except Exception:
            self.ok = False

    def _loop(self):
        c = ctypes.c_uint()
        r = ctypes.c_ulonglong()
        while not self._stop.is_set():
            if self.nv.nvmlDeviceGetClockInfo(self.h, 1, ctypes.byref(c)) == 0:
                rv = int(r.value) if self._reasons_fn(self.h, ctypes.byref(r)) == 0 else 0
                self.samples.append((int(c.value), rv))
            time.sleep(self.period)

    def start(self):
        if self.ok:
            self._stop.clear()
            self._thread = threading.Thread(target=self._loop, daemon=True)
            self._thread.start()

    def stop(self):
        if self._thread is not None:
            self._stop.set()
            self._thread.join()
        if not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": self.max_mhz, "reasons": [], "samples": 0,
                    "source": "nvml" if self.ok else "unavailable"}
        mhz = [s[0] for s in self.samples]
        bits = 0
        for _, rv in self.samples:
            bits |= rv
        reasons = [n for b, n in _REASONS.items() if bits & b]
        bins = {}
        for m in mhz:
            bins[str(m)] = bins.get(str(m), 0) + 1
        return {"sm_mhz": statistics.median(mhz), "sm_max_mhz": self.max_mhz,
                "sm_mhz_min": min(mhz), "reasons": reasons, "samples": len(mhz),
                "samples_by_sm_mhz": bins, "period_ms": self.period * 1e3, "source": "nvml"}


# ---------------------------------------------------------------------------
# Timed region: blocks of exactly K steps, repeated back to back
# ---------------------------------------------------------------------------

MIN_REGION_MS = 200.0


def timed_blocks(run_step, K, stream, first=0, min_ms=MIN_REGION_MS):
    """Time blocks of exactly K steps back to back on `stream` until the region covers
    `min_ms`, with a CUDA event between consecutive blocks.  run_step(i) enqueues step i.
    Returns (per-block ms, region ms, next step index, host us per step).  The caller
    brackets the call with its barrier and synchronisation."""
    import torch
    # pilot block (not part of the region) sizes the number of blocks
    p0 = torch.cuda.Event(enable_timing=True)
    p1 = torch.cuda.Event(enable_timing=True)
    p0.record(stream)
    for i in range(K):
        run_step(first + i)
    p1.record(stream)
    torch.cuda.synchronize()
    i0 = first + K
    est = max(p0.elapsed_time(p1), 1e-3)
    # a quarter more blocks than the pilot suggests (a warm block is shorter than the pilot)
    n_blocks = max(1, min(100000, int(-(-1.25 * min_ms // est)) + 1))
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(n_blocks + 1)]
    h0 = time.perf_counter()
    evs[0].record(stream)
    for b in range(n_blocks):
        for i in range(K):
            run_step(i0 + b * K + i)
        evs[b + 1].record(stream)
    h1 = time.perf_counter()
    torch.cuda.synchronize()
    blocks = [evs[b].elapsed_time(evs[b + 1]) for b in range(n_blocks)]
    return blocks, evs[0].elapsed_time(evs[-1]), i0 + n_blocks * K, (h1 - h0) * 1e6 / (n_blocks * K)


def block_stats(blocks, K):
    per = sorted(b / K for b in blocks)
    return {"blocks": len(blocks), "steps_per_block": K,
            "median_ms_per_step": statistics.median(per), "min_ms_per_step": per[0],
            "max_ms_per_step": per[-1], "mean_ms_per_step": sum(per) / len(per)}


# ---------------------------------------------------------------------------
# Peaks and ncu-derived traffic
# ---------------------------------------------------------------------------

def hbm_peak():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as fh:
            d = json.load(fh)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


# The sources that define the dominant kernel of the decode step (the tensor-core prefix
# kernel, its tcgen05 / TMA helpers, the branch/merge task it can run, and the descriptors
# both read).
TRAFFIC_SOURCES = ("pad_internal.h", "pad_tc_common.cuh", "pad_branch_merge.cuh", "pad_prefix_tc.cu")


def kernel_source_hash():
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2607_02963_gb300", "csrc")
    for f in TRAFFIC_SOURCES:
        with open(os.path.join(csrc, f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def recorded_traffic(workload, kernel):
    """dram read+write bytes per launch from the committed ncu summary, if it was taken
    on the current kernel sources for this workload; else None."""
    p = os.path.join(ROOT, "profiles", "prefix_traffic.txt")
    if not os.path.exists(p):
        return None
    want = kernel_source_hash()
    for line in open(p):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        kv = dict(x.split("=", 1) for x in line.split() if "=" in x)
        if kv.get("workload") == workload and kv.get("kernel") == kernel and kv.get("src") == want:
            return int(float(kv["dram_bytes_per_launch"]))
    return None


# ---------------------------------------------------------------------------
# CPU baseline: the fp64 oracle on a bounded sample
# ---------------------------------------------------------------------------

def blas_threads():
    try:
        from threadpoolctl import threadpool_info
        n = [i.get("num_threads") for i in threadpool_info() if i.get("user_api") == "blas"]
        if n:
            return int(max(n))
    except Exception:
        pass
    env = os.environ.get("OPENBLAS_NUM_THREADS") or os.environ.get("OMP_NUM_THREADS")
    return int(env) if env else os.cpu_count()


class OracleSample:
    """The fp64 oracle, as it stands, on (event, q-heads) samples of a workload.  The bf16
    inputs are widened to fp64 once, outside any timed region (the GPU arm likewise
    starts with its inputs resident)."""

    def __init__(self, w):
        import oracle
        self.oracle = oracle
        self.w = w
        f = oracle.bf16_to_f64
        self.kp = [f(w.prefix_k(b)) for b in range(w.n_videos)]
        self.vp = [f(w.prefix_v(b)) for b in range(w.n_videos)]
        self.q = f(w.q)
        self.kb = [np.concatenate([f(w.priv_k(e)), f(w.k_new[e:e + 1])]) for e in range(w.n_events)]
        self.vb = [np.concatenate([f(w.priv_v(e)), f(w.v_new[e:e + 1])]) for e in range(w.n_events)]

    def run(self, e, heads=None):
        """Oracle for event e (all heads, or the listed q-heads); returns event-tokens done."""
        b = int(self.w.event_video[e])
        self.oracle.video_attention(self.q[e:e + 1], self.kp[b], self.vp[b], [self.kb[e]],
                                    [self.vb[e]], self.w.scale, heads=heads)
        return 1.0 if heads is None else len(heads) / self.w.h_q


def cpu_baseline(w, budget_s=10.0):
    """Oracle, as it stands, on whole events of the workload until ~budget_s of CPU work."""
    smp = OracleSample(w)
    t0 = time.perf_counter()
    n = 0
    while True:  # whole events, cycling over the workload until the budget is spent
        smp.run(n % w.n_events)
        n += 1
        if time.perf_counter() - t0 >= budget_s and n >= min(w.n_events, 1):
            break
    dt = time.perf_counter() - t0
    return {"value": n / dt, "unit": UNIT, "cores": blas_threads(), "kind": "oracle",
            "sample": f"{n} event decodes ({n / w.n_events:.1f} passes over the {w.n_events} events "
                      f"of the workload; all {w.h_q} q-heads each; numpy fp64 with the explicit "
                      f"event mask; inputs widened to fp64 before timing), {dt:.1f} s"}


# ---------------------------------------------------------------------------
# GPU arm
# ---------------------------------------------------------------------------

def e2e_breakdown(step, run, n=200):
    """Where an end-to-end step's time goes: the library's own per-phase profile of
    pad_step_run_host (CUDA events between the phases on the step's stream, host clock
    readings beside them), means over n calls in microseconds."""
    step.profile(True)
    for i in range(n):
        run(i)
    d = step.profile_read()
    step.profile(False)
    d["how"] = ("pad_step_profile: events before the input copy, after it, after pad_plan, after "
                "the launches and after the output copy; host clock beside each; means")
    return d


def run_ours(args):
    import numpy as np
    import torch

    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    init_dist("nccl")

    from paper_2607_02963_gb300 import binding as B
    from paper_2607_02963_gb300 import build as pad_build
    from paper_2607_02963_gb300 import synth
    from paper_2607_02963_gb300.device import DeviceBatch, bits_to_bf16

    if rank == 0 or world == 1:
        pad_build.build()
    barrier(device)
    B.lib()

    w = make_workload(args.workload)
    byt = w.bytes_algorithmic()
    l2 = int(getattr(torch.cuda.get_device_properties(device), "L2_cache_size", 0) or (126 << 20))
    stream = torch.cuda.current_stream(device)

    flags = {"auto": 0, "simt": B.FLAG_PREFIX_SIMT, "mma": B.FLAG_PREFIX_MMA,
             "tc": B.FLAG_PREFIX_TC, "dual": B.FLAG_PREFIX_DUAL}[args.prefix]
    if args.fused_merge:
        flags |= B.FLAG_FUSED_MERGE
    first = DeviceBatch(w, device=device, fill_nan=False, flags=flags)
    per_rep = sum(t.numel() * t.element_size() for t in
                  (first.k_prefix, first.v_prefix, first.k_pool, first.v_pool, first.q, first.k_new,
                   first.v_new, first.out, first.lse, first.workspace, first.page_table))
    n_rep = args.replicas or max(2, -(-3 * l2 // per_rep))
    reps = [first] + [DeviceBatch(w, device=device, fill_nan=False, flags=flags)
                      for _ in range(n_rep - 1)]

    rope = self_g = None
    if args.rope:
        pos = synth.step_positions(w)
        rope = (pos, torch.from_numpy(synth.rope_table(int(pos.max()) + 1, w.head_dim)).to(device))
    if args.self_g:
        Kp = np.array([min(int(w.prefix_len[b]) - 1, len(w.events_of_video(b)) + 2)
                       for b in range(w.n_videos)], np.int32)
        gi = np.zeros(w.n_events, np.int32)
        for b in range(w.n_videos):
            ev = w.events_of_video(b)
            if Kp[b] > 0:
                gi[ev] = np.arange(len(ev)) % Kp[b]
        self_g = (Kp, gi)

    # the library's step executor: one C call per step (pad_step_run), or with the host
    # copies and the wait included (pad_step_run_host)
    def launcher(db, **kw):
        return B.NativeStep(db.problem, db.cache, w.prefix_len, w.event_video, w.event_len,
                            db.page_table, w.max_pages, db.workspace, w.prefix_offset,
                            kw.get("q", db.q), db.k_new, db.v_new, db.k_prefix, db.v_prefix,
                            db.k_pool, db.v_pool, db.out, db.lse, kw.get("stream", stream),
                            one_call=not args.two_call, rope=rope, self_g=self_g, causal=args.causal,
                            mapped_host_io=kw.get("mapped", not args.e2e_copy))

    one_call = not args.two_call
    api_path = ("pad_step_run (pad_plan + pad_decode_step)" if one_call
                else "pad_step_run (pad_plan + pad_kv_append + pad_event_decode_attn)")
    steps = [launcher(db) for db in reps]
    info = reps[0].plan_step(stream).info()
    # kernels of one step: append (two-call path only), prefix pass, branch/merge (unless
    # the prefix kernel runs it)
    launches_per_step = ((0 if one_call else 1) + (info["n_work_items"] > 0)
                         + (0 if info["fused_tail"] else 1))
    reps[0].release_new_pages()
    torch.cuda.synchronize()

    W, K = max(3, args.warmup), args.steps
    for i in range(W):
        steps[i % n_rep]()
    torch.cuda.synchronize()
    for db in reps:  # a kernel-side error (e.g. a bounded wait that gave up) stops the run here
        B.pad_device_status(db.plan_step(stream))
        db.release_new_pages()
    barrier(device)
    if args.profile_run:
        # a short run for a profiler: the warm-up above, then exactly this many steps,
        # no timing loops (launch count = steps x kernels per step)
        for i in range(args.profile_run):
            steps[(W + i) % n_rep]()
        torch.cuda.synchronize()
        for db in reps:
            B.pad_device_status(db.plan_step(stream))
            db.release_new_pages()
        if rank == 0:
            print(json.dumps({"profile_run": args.profile_run, "warmup": W, "workload": args.workload,
                              "kernels_per_step": launches_per_step, "replicas": n_rep}), flush=True)
        return

    # timed region: blocks of exactly K steps, each step exactly as a caller runs it (no
    # events between its kernels, an event between blocks), repeated to cover >= 200 ms
    sampler = ClockSampler(local)
    barrier(device)
    torch.cuda.synchronize()
    sampler.start()
    blocks, region_ms, nxt, host_us = timed_blocks(lambda i: steps[(W + i) % n_rep](), K, stream)
    torch.cuda.synchronize()
    barrier(device)
    clocks = sampler.stop()
    bstat = block_stats(blocks, K)
    ms = bstat["median_ms_per_step"] * K
    # the shared-prefix kernel alone: CUDA events around each of its launches (the
    # library records them on the launching stream; overlap with neighbours is off)
    Kr = max(K, 500)
    B.pad_timing_enable(Kr)
    for i in range(Kr):
        steps[(W + nxt + i) % n_rep]()
    torch.cuda.synchronize()
    pre_ms, pre_n = B.pad_timing_read()
    for db in reps:
        B.pad_device_status(db.plan_step(stream))
        db.release_new_pages()

    units, ms_max = aggregate(float(w.n_events * K), ms, device)
    value = units / (ms_max * 1e-3)

    # e2e through the C ABI with host buffers: H2D inputs, step, D2H outputs, sync.
    Ke = max(3, min(K, args.e2e_steps))
    # page-locked host buffers laid out like the device ones (q | k_new | v_new, out | lse)
    h_in = torch.empty(reps[0].io_in.shape, dtype=torch.bfloat16, pin_memory=True)
    h_out = torch.empty(reps[0].io_out.shape, dtype=torch.uint8, pin_memory=True)
    qn, kn = w.q.size, w.k_new.size
    hq = h_in[:qn].view(reps[0].q.shape)
    hkn = h_in[qn:qn + kn].view(reps[0].k_new.shape)
    hvn = h_in[qn + kn:].view(reps[0].v_new.shape)
    hq.copy_(bits_to_bf16(w.q, "cpu"))
    hkn.copy_(bits_to_bf16(w.k_new, "cpu"))
    hvn.copy_(bits_to_bf16(w.v_new, "cpu"))
    ob = reps[0].out.numel() * reps[0].out.element_size()
    hout = h_out[:ob].view(reps[0].out.dtype).view(reps[0].out.shape)
    hlse = h_out[ob:].view(torch.float32).view(reps[0].lse.shape)
    h2d = sum(t.numel() * t.element_size() for t in (hq, hkn, hvn))
    d2h = sum(t.numel() * t.element_size() for t in (hout, hlse))

    def e2e_blocks(run):
        for i in range(3):
            run(i)
        barrier(device)
        # blocks of Ke steps on the host clock until the region covers >= 200 ms
        blocks = []
        t_start = time.perf_counter()
        i = 0
        while True:
            t0 = time.perf_counter()
            for _ in range(Ke):
                run(i)
                i += 1
            t1 = time.perf_counter()
            blocks.append((t1 - t0) * 1e3)
            if (t1 - t_start) * 1e3 >= MIN_REGION_MS:
                return block_stats(blocks, Ke)

    # A second set of page-locked buffers for a second, independent batch (the next replica)
    h_in2 = torch.empty_like(h_in, pin_memory=True)
    h_out2 = torch.empty_like(h_out, pin_memory=True)
    h_in2.copy_(h_in)
    io = [(hq, hkn, hvn, hout, hlse),
          (h_in2[:qn].view(hq.shape), h_in2[qn:qn + kn].view(hkn.shape), h_in2[qn + kn:].view(hvn.shape),
           h_out2[:ob].view(hout.dtype).view(hout.shape), h_out2[ob:].view(torch.float32).view(hlse.shape))]
    # the second batch on a stream of its own (--e2e-streams 2), so that one batch's host
    # reads and writes and its merge tail can overlap the other batch's kernels
    stream2 = torch.cuda.Stream(device) if args.e2e_streams > 1 else stream
    pair = [steps[0], launcher(reps[1 % n_rep], stream=stream2) if args.e2e_streams > 1 else steps[1 % n_rep]]

    def pipelined_block(n):
        # two batches in flight: batch i % 2 is planned and enqueued (pad_step_enqueue_host)
        # while the device runs batch (i - 1) % 2, whose outputs the host then waits for
        pair[0].enqueue_host(*io[0])
        for i in range(1, n):
            pair[i % 2].enqueue_host(*io[i % 2])
            pair[(i - 1) % 2].wait()
        pair[(n - 1) % 2].wait()

    def e2e_blocks(run_block):
        run_block(3)
        barrier(device)
        # blocks of Ke steps on the host clock until the region covers >= 200 ms
        blocks = []
        t_start = time.perf_counter()
        while True:
            t0 = time.perf_counter()
            run_block(Ke)
            t1 = time.perf_counter()
            blocks.append((t1 - t0) * 1e3)
            if (t1 - t_start) * 1e3 >= MIN_REGION_MS:
                return block_stats(blocks, Ke)

    def serial_block(st):
        def run(n):
            for i in range(n):
                st.run_host(hq, hkn, hvn, hout, hlse)
        return run

    mapped = not args.e2e_copy
    io_desc = (("q/k_new/v_new read from pinned mapped host memory by a kernel, " if mapped
                else "pinned H2D copy of q/k_new/v_new, ")
               + "pad_plan + " + ("pad_decode_step" if one_call else "pad_kv_append + pad_event_decode_attn")
               + (", O and LSE written into pinned mapped host memory by the step's kernels" if mapped
                  else ", D2H copy of O and LSE"))
    # headline: two independent batches in flight through pad_step_enqueue_host / pad_step_wait
    e_stat = e2e_blocks(pipelined_block)
    e_units, e_ms = aggregate(float(w.n_events * Ke), e_stat["median_ms_per_step"] * Ke, device)
    e2e = {"value": e_units / (e_ms * 1e-3), "unit": UNIT, "h2d_bytes_per_step": h2d,
           "d2h_bytes_per_step": d2h, "steps": Ke, "us_per_step": e_stat["median_ms_per_step"] * 1e3,
           "in_flight": 2,
           "timing": dict(e_stat, clock="host perf_counter around each block of steps"),
           "path": "through the C ABI, every step: " + io_desc + "; two independent batches (own "
                   "executor, own host buffers" + (", own stream" if args.e2e_streams > 1 else ", one stream")
                   + ") in flight: pad_step_enqueue_host of one, then pad_step_wait of the other"}
    # one batch, each step waited for before the next (pad_step_run_host)
    s_stat = e2e_blocks(serial_block(steps[0]))
    e2e["serial"] = {"us_per_step": s_stat["median_ms_per_step"] * 1e3,
                     "value": w.n_events / s_stat["median_ms_per_step"] * 1e3,
                     "path": "pad_step_run_host, one batch: " + io_desc + ", stream wait, every step",
                     "breakdown_us": e2e_breakdown(steps[0], lambda i: steps[0].run_host(hq, hkn, hvn, hout, hlse))}
    if mapped:
        # the same serial call on the copy-engine path (cudaMemcpyAsync both ways)
        alt = launcher(reps[0], mapped=False)
        a_stat = e2e_blocks(serial_block(alt))
        e2e["serial_copy_engine"] = {
            "us_per_step": a_stat["median_ms_per_step"] * 1e3,
            "value": w.n_events / a_stat["median_ms_per_step"] * 1e3,
            "breakdown_us": e2e_breakdown(alt, lambda i: alt.run_host(hq, hkn, hvn, hout, hlse))}
        del alt

    if rank != 0:
        return
    peak, peak_kind = hbm_peak()
    kern_name = {1: "prefix_simt_kernel", 2: "prefix_mma_kernel", 4: "prefix_tc_kernel",
                 16: "prefix_dual_kernel"}[
        info["prefix_kernel"]]
    prefix_ms_per_launch = pre_ms / max(1, pre_n)
    # the timed kernel's own algorithmic bytes: the prefix pass alone, or, when it also runs
    # a4 + a5 (and a2 in the one-call step), every byte of the step that it moves
    fused = bool(info["fused_tail"])
    if fused:
        roof_bytes = byt["total"] - (0 if one_call else byt["append"])
        roof_what = "prefix + branch KV + Q + out/LSE" + (" + append" if one_call else "")
    else:
        roof_bytes = byt["prefix"]
        roof_what = "prefix KV read once"
    achieved = roof_bytes / (prefix_ms_per_launch * 1e-3) / 1e9
    step_ms = ms / K
    line = {
        "metric": METRIC,
        "value": value,
        "unit": UNIT,
        "n_gpus": world,
        "steps": K,
        "warmup": W,
        "ms_per_step": ms_max / K,
        "timing": dict(bstat, region_ms=region_ms,
                       how="CUDA events on the launching stream between back-to-back blocks "
                           "of exactly K steps; value and ms_per_step from the median block"),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic: seeded N(0,1) bf16 Q/K/V shaped like the paper's long omni-modal "
                "videos (no dataset or weights)",
        "config": {
            "workload": args.workload,
            "description": WORKLOADS[args.workload],
            "videos": w.n_videos, "events": w.n_events, "h_q": w.h_q, "h_kv": w.h_kv,
            "head_dim": w.head_dim, "page_size": w.page_size,
            "prefix_tokens": int(w.prefix_len.sum()),
            "private_tokens_after_append": int((w.event_len + 1).sum()),
            "prefix_kernel": kern_name, "splits": info["n_work_items"],
            "fused_tail": bool(info["fused_tail"]), "api": api_path,
            "variants": {"rope": bool(args.rope), "self_g_only": bool(args.self_g),
                         "causal": bool(args.causal)},
            "l2": f"{n_rep} rotating cold replicas of the whole device state "
                  f"({n_rep * per_rep / 2**20:.0f} MiB > 3x L2 {l2 / 2**20:.0f} MiB)",
            "parallelism": "replicas" if world > 1 else "single GPU",
        },
        "clocks": clocks,
        "gpu_launches": K * launches_per_step,
        "roofline": {
            "bound": "hbm",
            "kernel": kern_name,
            "achieved": achieved,
            "peak": peak,
            "unit": "GB/s",
            "frac": achieved / peak,
            "peak_kind": peak_kind,
            "traffic": recorded_traffic(args.workload, kern_name),
            "algorithmic_bytes_per_launch": roof_bytes,
            "algorithmic_bytes_cover": roof_what,
            "fused_tail": fused,
            "launch_us": prefix_ms_per_launch * 1e3,
            "launches_timed": pre_n,
            "timing": "CUDA events around each launch of the kernel on its stream, in a loop of "
                      "full steps after the timed one",
        },
        "step": {
            "us": step_ms * 1e3,
            "algorithmic_bytes": byt["total"],
            "achieved_gbs": byt["total"] / (step_ms * 1e-3) / 1e9,
            "frac_of_measured_hbm": byt["total"] / (step_ms * 1e-3) / 1e9 / peak,
            "frac_of_nominal_8tbs": byt["total"] / (step_ms * 1e-3) / 1e9 / 8000.0,
            "host_us_per_step": host_us,
        },
        "e2e": e2e,
    }
    if not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(w, args.cpu_budget)
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------------------
# Reference arm: the fp64 oracle on the host cores
# ---------------------------------------------------------------------------

def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return
    w = make_workload(args.workload)
    H = w.h_q
    smp = OracleSample(w)
    # size each step's sample (q-head rows of one event) so the run stays within ~120 s
    t0 = time.perf_counter()
    smp.run(0, [0])
    t_row = max(time.perf_counter() - t0, 1e-4)
    total = args.steps + max(3, args.warmup)
    rows_per_step = int(max(1, min(H, 120.0 / (total * t_row))))

    def step(i):
        e = i % w.n_events
        h0 = (i * rows_per_step) % H
        return smp.run(e, [(h0 + j) % H for j in range(rows_per_step)])

    W, K = max(3, args.warmup), args.steps
    for i in range(W):
        step(i)
    t0 = time.perf_counter()
    done = 0.0
    for i in range(K):
        done += step(W + i)
    dt = time.perf_counter() - t0
    value = done / dt
    line = {
        "impl": "reference",
        "metric": METRIC,
        "value": value,
        "unit": UNIT,
        "n_gpus": world,
        "steps": K,
        "warmup": W,
        "ms_per_step": dt * 1e3 / K,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "f64",
        "data": "synthetic: seeded N(0,1) bf16 Q/K/V widened exactly to fp64",
        "config": {"workload": args.workload, "description": WORKLOADS[args.workload],
                   "videos": w.n_videos, "events": w.n_events, "h_q": w.h_q, "h_kv": w.h_kv,
                   "head_dim": w.head_dim, "prefix_tokens": int(w.prefix_len.sum()),
                   "parallelism": "host cores"},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": blas_threads(), "kind": "oracle",
                         "sample": f"{rows_per_step} q-head row(s) of one event of the workload per step "
                                   f"(numpy fp64, explicit event mask, inputs widened to fp64 "
                                   f"before timing)"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def run_prefill(args):
    """Whole-sequence forward attention under the event-factorized mask (training /
    prefill), on the long_32k video: prefix 32768 tokens, then its 32 branches (each the
    branch's tokens after this step, 1917 in all).  Timed with CUDA events over repeated
    calls (compute-bound; inputs stay resident).  Comparators on the same tensors: torch's
    scaled_dot_product_attention with the explicit boolean mask (the generic masked path the
    paper used), and with is_causal=True (the plain causal kernel, which computes a
    different mask: a speed reference only)."""
    import math
    import numpy as np
    import torch
    import torch.nn.functional as F
    from paper_2607_02963_gb300 import binding as B
    from paper_2607_02963_gb300 import build as pad_build
    from paper_2607_02963_gb300 import synth

    device = torch.device("cuda", 0)
    torch.cuda.set_device(device)
    pad_build.build()
    B.lib()
    w = synth.long_32k()
    S = int(w.prefix_len[0])
    lens = (w.event_len + 1).astype(np.int32)
    H, Hkv, D = w.h_q, w.h_kv, w.head_dim
    qb, kb, vb = synth.prefill_inputs(11, S, lens, H, Hkv, D, k_scale_sigma=0.5)
    N = qb.shape[0]

    def dev(bits):
        return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).to(device)

    q, k, v = dev(qb), dev(kb), dev(vb)
    out = torch.empty((N, H, D), dtype=torch.float32, device=device)
    lse = torch.empty((N, H), dtype=torch.float32, device=device)
    prob = B.make_problem(H, Hkv, D, 16, 1.0 / math.sqrt(D))
    stream = torch.cuda.current_stream(device)

    def timed(fn, n):
        for _ in range(2):
            fn()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(n):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / n

    K = max(3, min(args.steps, 20))
    ms = timed(lambda: B.pad_prefill_attn(prob, S, lens, q, k, v, out, lse, stream), K)
    B.pad_prefill_status(stream)
    prob_mma = B.make_problem(H, Hkv, D, 16, 1.0 / math.sqrt(D), flags=B.FLAG_PREFIX_MMA)
    mma_ms = timed(lambda: B.pad_prefill_attn(prob_mma, S, lens, q, k, v, out, lse, stream), max(2, K // 4))
    # visible (query, key) pairs: the prefix's causal triangle, plus every branch token's
    # prefix and its own earlier branch tokens
    pairs = S * (S + 1) // 2 + sum(int(n) * S + int(n) * (int(n) + 1) // 2 for n in lens)
    flops = 4.0 * pairs * D * H
    peak = 1862.7
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as fh:
            peak = float(json.load(fh)["bf16_tflops"])
        peak_kind = "measured"
    except Exception:
        peak_kind = "fallback"
    qt = q.permute(1, 0, 2).unsqueeze(0)
    kt = k.permute(1, 0, 2).repeat_interleave(H // Hkv, dim=0).unsqueeze(0)
    vt = v.permute(1, 0, 2).repeat_interleave(H // Hkv, dim=0).unsqueeze(0)
    causal_ms = timed(lambda: F.scaled_dot_product_attention(qt, kt, vt, is_causal=True), K)
    masked_ms = None
    try:
        starts = np.concatenate([[S], S + np.cumsum(lens)[:-1]])
        pos = torch.arange(N, device=device)
        br = torch.full((N,), -1, dtype=torch.long, device=device)
        for b, (st, n) in enumerate(zip(starts, lens)):
            br[int(st):int(st) + int(n)] = b
        mask = (pos[None, :] <= pos[:, None]) & ((pos[None, :] < S) | (br[None, :] == br[:, None]))
        masked_ms = timed(lambda: F.scaled_dot_product_attention(qt, kt, vt, attn_mask=mask), max(2, K // 4))
        del mask
    except Exception as ex:  # noqa: BLE001 - the comparator is optional
        masked_ms = f"unavailable: {type(ex).__name__}"
    line = {
        "metric": "prefill_tokens_per_s", "value": N / (ms * 1e-3), "unit": "tokens/s",
        "higher_is_better": True, "n_gpus": 1, "steps": K, "warmup": 2, "dtype": "bf16 in, fp32 accumulate",
        "data": "synthetic: seeded N(0,1) bf16 q/k/v of the long_32k video's whole sequence",
        "config": {"workload": "prefill_long_32k", "prefix_tokens": S, "branches": int(lens.size),
                   "branch_tokens": int(lens.sum()), "tokens": N, "h_q": H, "h_kv": Hkv, "head_dim": D,
                   "kernel": "prefix_tc_kernel (tcgen05, prefill mode)"},
        "ms": ms,
        "roofline": {"bound": "tensor", "achieved": flops / (ms * 1e-3) / 1e12, "peak": peak, "unit": "TFLOP/s",
                     "frac": flops / (ms * 1e-3) / 1e12 / peak, "peak_kind": peak_kind,
                     "flops": flops, "visible_pairs_per_head": pairs},
        "comparators_ms": {"torch_sdpa_explicit_mask": masked_ms, "torch_sdpa_is_causal": causal_ms,
                           "ours_mma_sync_kernel": mma_ms},
        "gpu_launches": K,
    }
    print(json.dumps(line), flush=True)


def run_grounding(args):
    """Grounding readout of the long_32k video (Sec. 3.3): segment pooling of the projected
    prefix, scoring of the 32 event tokens, attention-guided aggregation; each kernel timed
    with CUDA events over rotating input replicas larger than L2."""
    import numpy as np
    import torch
    from paper_2607_02963_gb300 import binding as B
    from paper_2607_02963_gb300 import build as pad_build
    from paper_2607_02963_gb300 import synth

    device = torch.device("cuda", 0)
    torch.cuda.set_device(device)
    pad_build.build()
    B.lib()
    T, S, K, dp, dm = 32768, 128, 32, 256, 2048
    gi = synth.grounding_inputs(3, T, S, K, dp, dm, text_tokens=32)

    def dev(bits):
        return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).to(device)

    l2 = int(getattr(torch.cuda.get_device_properties(device), "L2_cache_size", 0) or (126 << 20))
    f0, x0 = dev(gi.f_proj), dev(gi.x)
    nf = max(2, -(-3 * l2 // (f0.numel() * 2)))
    nx = max(2, -(-3 * l2 // (x0.numel() * 2)))
    fs = [f0] + [f0.clone() for _ in range(nf - 1)]
    xs = [x0] + [x0.clone() for _ in range(nx - 1)]
    g, emb = dev(gi.g_proj), dev(gi.g_emb)
    attn = torch.from_numpy(gi.attn).to(device)
    seg = torch.empty((S, dp), dtype=torch.float32, device=device)
    sc = torch.empty((K, S), dtype=torch.float32, device=device)
    sal = torch.empty((K, S), dtype=torch.uint8, device=device)
    iv = torch.empty((K, 2), dtype=torch.int32, device=device)
    out = torch.empty((K, dm), dtype=torch.float32, device=device)
    ws = B.aggregate_workspace(T, S, dm, device)
    stream = torch.cuda.current_stream(device)
    W, N = max(3, args.warmup), max(10, min(args.steps, 500))

    # The calls are captured in a CUDA graph (20 per graph, over the rotating replicas) and
    # the graph is replayed: the kernels' time, not the Python calls' (a few times longer).
    G = 20

    def timed(fn):
        for i in range(W):
            fn(i, stream)
        torch.cuda.synchronize()
        cap = torch.cuda.Stream(device)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=cap):
            for i in range(G):
                fn(i, cap)
        reps = max(1, N // G)
        for _ in range(2):
            graph.replay()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(reps):
            graph.replay()
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) * 1e3 / (reps * G)

    pool_us = timed(lambda i, s: B.pad_ground_pool(fs[i % nf], gi.offsets, seg, s))
    score_us = timed(lambda i, s: B.pad_ground_score(g, seg, 0.5, sc, sal, iv, s))
    agg_us = timed(lambda i, s: B.pad_attn_aggregate(xs[i % nx], attn, gi.offsets, iv, emb, out, ws, s))

    def whole(i, s):
        B.pad_ground_pool(fs[i % nf], gi.offsets, seg, s)
        B.pad_ground_score(g, seg, 0.5, sc, sal, iv, s)
        B.pad_attn_aggregate(xs[i % nx], attn, gi.offsets, iv, emb, out, ws, s)

    all_us = timed(whole)
    ivh = iv.cpu().numpy()
    tok = sum(int(gi.offsets[ivh[i, 1] + 1] - gi.offsets[ivh[i, 0]]) for i in range(K))
    # the events' intervals overlap: a hidden-state row that several events aggregate needs
    # to come from HBM once, so the algorithmic bytes count the distinct rows
    covered = np.zeros(T, dtype=bool)
    for i in range(K):
        covered[int(gi.offsets[ivh[i, 0]]):int(gi.offsets[ivh[i, 1] + 1])] = True
    distinct = int(covered.sum())
    peak, peak_kind = hbm_peak()
    pool_bytes = T * dp * 2 + S * dp * 4
    agg_bytes = distinct * dm * 2 + tok * 4 + K * dm * (2 + 4)
    line = {
        "metric": "grounding_readouts_per_s", "value": 1e6 / all_us, "unit": "video readouts/s",
        "higher_is_better": True, "n_gpus": 1, "steps": N, "warmup": W, "dtype": "bf16 in, fp32 accumulate",
        "data": "synthetic: seeded projected features and hidden states shaped like the long_32k video",
        "config": {"workload": "grounding_long_32k", "prefix_tokens": T, "segments": S, "events": K,
                   "d_proj": dp, "d_model": dm, "fraction": 0.5, "grounded_tokens": tok, "distinct_grounded_tokens": distinct,
                   "l2": f"{nf} / {nx} rotating replicas of the projected features / hidden states (> 3x L2)"},
        "us": {"pool": pool_us, "score": score_us, "aggregate": agg_us, "readout": all_us},
        "roofline": {
            "pool": {"bound": "hbm", "bytes": pool_bytes, "achieved": pool_bytes / pool_us / 1e3, "peak": peak,
                     "unit": "GB/s", "frac": pool_bytes / pool_us / 1e3 / peak, "peak_kind": peak_kind},
            "aggregate": {"bound": "hbm", "bytes": agg_bytes, "achieved": agg_bytes / agg_us / 1e3, "peak": peak,
                          "unit": "GB/s", "frac": agg_bytes / agg_us / 1e3 / peak, "peak_kind": peak_kind},
        },
        "gpu_launches": 3 * G * max(1, N // G),
        "timing": "CUDA events around replays of a CUDA graph of 20 calls per kernel (and of 20 readouts)",
    }
    print(json.dumps(line), flush=True)


def run_sweep(args):
    """Per E: our step (cold replicas, back to back) and the naive per-event comparator."""
    import torch
    import torch.nn.functional as F
    from paper_2607_02963_gb300 import binding as B
    from paper_2607_02963_gb300 import build as pad_build
    from paper_2607_02963_gb300.device import DeviceBatch

    device = torch.device("cuda", 0)
    torch.cuda.set_device(device)
    pad_build.build()
    B.lib()
    stream = torch.cuda.current_stream(device)
    l2 = int(getattr(torch.cuda.get_device_properties(device), "L2_cache_size", 0) or (126 << 20))
    flush = torch.empty(3 * l2, dtype=torch.uint8, device=device)
    peak, peak_kind = hbm_peak()
    for E in (1, 2, 4, 8, 16, 32, 64):
        w = make_workload(f"sweep_e{E}")
        byt_all = w.bytes_algorithmic()
        byt = byt_all["total"]
        first = DeviceBatch(w, device=device, fill_nan=False)
        per_rep = first.k_prefix.numel() * 4 + first.k_pool.numel() * 4
        n_rep = max(2, -(-3 * l2 // per_rep))
        reps = [first] + [DeviceBatch(w, device=device, fill_nan=False) for _ in range(n_rep - 1)]
        steps = [B.NativeStep(db.problem, db.cache, w.prefix_len, w.event_video, w.event_len,
                                db.page_table, w.max_pages, db.workspace, w.prefix_offset, db.q,
                                db.k_new, db.v_new, db.k_prefix, db.v_prefix, db.k_pool, db.v_pool,
                                db.out, db.lse, stream) for db in reps]
        W = max(3, args.warmup)
        for i in range(W):
            steps[i % n_rep]()
        torch.cuda.synchronize()
        K = args.steps
        sampler = ClockSampler(0)
        sampler.start()
        blocks, region_ms, nxt, _ = timed_blocks(lambda i: steps[(W + i) % n_rep](), K, stream)
        clocks = sampler.stop()
        bstat = block_stats(blocks, K)
        ours_us = bstat["median_ms_per_step"] * 1e3
        B.pad_timing_enable(500)
        for i in range(500):
            steps[(W + nxt + i) % n_rep]()
        torch.cuda.synchronize()
        pre_ms, pre_n = B.pad_timing_read()
        pre_us = pre_ms * 1e3 / max(1, pre_n)
        for db in reps:
            B.pad_device_status(db.plan_step(stream))
            db.release_new_pages()

        # naive comparator: per event, its visible keys made contiguous once (outside the
        # timing), then one attention call per event per step; L2 flushed between steps
        db = first
        steps[0]()
        torch.cuda.synchronize()
        ks, vs, qs = [], [], []
        for e in range(w.n_events):
            b_ = int(w.event_video[e])
            o, P = int(w.prefix_offset[b_]), int(w.prefix_len[b_])
            kb, vb = db.gather_branch(e, int(w.event_len[e]) + 1)
            ks.append(torch.cat([db.k_prefix[o:o + P], kb]).transpose(0, 1).unsqueeze(0).contiguous())
            vs.append(torch.cat([db.v_prefix[o:o + P], vb]).transpose(0, 1).unsqueeze(0).contiguous())
            qs.append(db.q[e].view(1, w.h_q, 1, w.head_dim))
        naive_bytes = sum(k.numel() * 2 * 2 for k in ks)
        outs = [None] * w.n_events
        times = []
        for it in range(3 + args.sweep_naive_steps):
            flush.zero_()
            a0 = torch.cuda.Event(enable_timing=True)
            a1 = torch.cuda.Event(enable_timing=True)
            a0.record(stream)
            for e in range(w.n_events):
                outs[e] = F.scaled_dot_product_attention(qs[e], ks[e], vs[e], scale=float(w.scale),
                                                         enable_gqa=True)
            a1.record(stream)
            torch.cuda.synchronize()
            if it >= 3:
                times.append(a0.elapsed_time(a1) * 1e3)
        naive_us = statistics.median(times)
        ref = torch.stack([o.view(w.h_q, w.head_dim).float() for o in outs])
        diff = float((ref - db.out.float()).abs().max())
        gbs = byt / ours_us * 1e-3
        print(json.dumps({
            "metric": METRIC, "value": w.n_events / (ours_us * 1e-6), "unit": UNIT,
            "sweep_E": E, "workload": f"sweep_e{E}", "description": WORKLOADS[f"sweep_e{E}"],
            "algorithmic_bytes": byt, "prefix_bytes": byt_all["prefix"], "branch_bytes": byt_all["branch"],
            "ours_us_per_step": ours_us, "ours_min_us_per_step": bstat["min_ms_per_step"] * 1e3,
            "ours_gbs": gbs, "frac_of_measured_hbm": gbs / peak, "peak_gbs": peak, "peak_kind": peak_kind,
            "prefix_kernel_us": pre_us, "prefix_kernel_frac": byt_all["prefix"] / pre_us * 1e-3 / peak,
            "naive_bytes_per_step": naive_bytes, "naive_us_per_step": naive_us,
            "naive_gbs": naive_bytes / naive_us * 1e-3, "naive_over_ours_time": naive_us / ours_us,
            "max_abs_ours_vs_naive": diff, "replicas": n_rep,
            "timing": dict(bstat, region_ms=region_ms), "clocks": clocks}), flush=True)
        del reps, steps, first, db, ks, vs, qs, outs
        torch.cuda.empty_cache()


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", choices=sorted(WORKLOADS), default="long_32k")
    ap.add_argument("--replicas", type=int, default=0, help="cold replicas (0 = enough for 3x L2)")
    ap.add_argument("--prefix", choices=["auto", "simt", "mma", "tc", "dual"], default="auto",
                    help="shared-prefix kernel (auto = the library's choice)")
    ap.add_argument("--e2e-steps", type=int, default=500)
    ap.add_argument("--e2e-streams", type=int, default=2, choices=(1, 2),
                    help="streams of the two batches in flight in the headline e2e measurement")
    ap.add_argument("--e2e-copy", action="store_true",
                    help="e2e through the copy-engine path of pad_step_run_host (no mapped host I/O)")
    ap.add_argument("--cpu-budget", type=float, default=10.0, help="seconds of oracle work")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--fused-merge", action="store_true",
                    help="a4 + a5 inside the tensor-core prefix kernel where the plan allows it")
    ap.add_argument("--prefill", action="store_true",
                    help="time the whole-sequence masked attention (training / prefill) of the long_32k video")
    ap.add_argument("--grounding", action="store_true",
                    help="time the grounding readout (pool, score, aggregate) of the long_32k video")
    ap.add_argument("--rope", action="store_true",
                    help="rotate q and k_new inside the step at the shared step position")
    ap.add_argument("--self-g", action="store_true",
                    help="the self G-token only mask (K = events + 2 planning tokens per video)")
    ap.add_argument("--causal", action="store_true", help="the causal-attention mask variant")
    ap.add_argument("--two-call", action="store_true",
                    help="pad_kv_append + pad_event_decode_attn instead of pad_decode_step")
    ap.add_argument("--sweep", action="store_true",
                    help="per-E table of the sweep workload with the naive per-event comparator")
    ap.add_argument("--sweep-naive-steps", type=int, default=20)
    ap.add_argument("--profile-run", type=int, default=0,
                    help="run the warm-up and then this many steps only (for ncu), no timing")
    args = ap.parse_args(argv)
    if args.prefill:
        run_prefill(args)
    elif args.grounding:
        run_grounding(args)
    elif args.sweep:
        run_sweep(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)
    try:
        import torch.distributed as dist
        if dist.is_initialized():
            dist.destroy_process_group()
    except Exception:
        pass


if __name__ == "__main__":
    main()
