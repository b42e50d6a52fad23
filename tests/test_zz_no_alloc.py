"""The allocation-free attention call, pad_event_decode_attn_static.

It exists for callers that cannot give the library device scratch memory (a plugin
interface that hands out tensors but no allocator, or a serving loop whose device memory
is fixed before it starts): the plan image and the split-KV partial states go to a 16 MiB
array inside the library instead of a caller workspace.  These tests check it against the
workspace path on the same step, twice in a row (the array keeps the previous call's
contents), and that plans too large for the array are refused before anything runs.
"""
import numpy as np
import pytest
import torch

from paper_2607_02963_gb300 import binding as B
from paper_2607_02963_gb300 import synth
from paper_2607_02963_gb300.device import DeviceBatch

MAX_ABS = 1e-2
REL_L2 = 2e-3
LSE_ABS = 1e-3


def test_plans_larger_than_the_static_array_are_refused(padlib):
    # 16 videos x 64 events x 16 query heads per kv-head: more partial states than 16 MiB hold
    prob = B.make_problem(64, 4, 128, num_sms=152)
    cache = B.CacheState(4096)
    ev = np.repeat(np.arange(16, dtype=np.int32), 64)
    plan = B.pad_plan(prob, cache, [8192] * 16, ev, np.ones(ev.size, dtype=np.int32), max_pages=2,
                      workspace=None)
    assert plan.info()["workspace_bytes"] > 16 << 20
    with pytest.raises(B.PadError) as ei:
        B._check(B.lib().pad_event_decode_attn_static(plan.handle, None, None, None, None, None,
                                                      None, None, None))
    assert ei.value.status == 4 and "static scratch" in str(ei.value)


def _compare(got_o, got_l, ref_o, ref_l):
    got = got_o.double().cpu().numpy()
    ref = ref_o.double().cpu().numpy()
    assert np.all(np.isfinite(got))
    assert np.abs(got - ref).max() <= MAX_ABS
    assert np.linalg.norm(got - ref) / np.linalg.norm(ref) <= REL_L2
    assert np.abs(got_l.double().cpu().numpy() - ref_l.double().cpu().numpy()).max() <= LSE_ABS


@pytest.mark.gpu
@pytest.mark.parametrize("make", [synth.gqa_8k, synth.tiny,
                                  lambda: synth.random_small(5, h_q=8, h_kv=2, max_events=3)])
def test_static_scratch_matches_workspace_path_twice(padlib, make):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    w = make()
    db = DeviceBatch(w)
    plan = db.run_step()                       # append + attention through the workspace
    torch.cuda.synchronize()
    B.pad_device_status(plan)
    ref_o, ref_l = db.out.clone(), db.lse.clone()
    # a host-only plan of the same step (no workspace): hand back the pages the first
    # plan took, so the allocation repeats exactly
    db.release_new_pages(plan)
    hplan = B.pad_plan(db.problem, db.cache, w.prefix_len, w.event_video, w.event_len,
                       page_table=db.page_table, max_pages=w.max_pages, workspace=None,
                       prefix_offset=w.prefix_offset)
    assert np.array_equal(hplan.new_pages(), plan.new_pages())
    for _ in range(2):
        o = torch.full_like(db.out, float("nan"))
        lse = torch.full_like(db.lse, float("nan"))
        B.pad_event_decode_attn_static(hplan, db.q, db.k_prefix, db.v_prefix, db.k_pool, db.v_pool,
                                       o, lse)
        torch.cuda.synchronize()
        _compare(o, lse, ref_o, ref_l)


# ---------------------------------------------------------------------------
# A whole decode loop with no device scratch: host-only plans for both calls
# ---------------------------------------------------------------------------

def _next_step(w, seed):
    """The workload of the following decode step: every branch one token longer (this step's
    new K/V appended), a fresh q / k_new / v_new, and the page table and free list as the
    step left them (the oracle's simulation of the append)."""
    import dataclasses
    import oracle
    st, pt, free, _ = oracle.simulate_append(w.page_table, w.free_pages, w.event_len, w.page_size)
    assert st == oracle.OK
    rng = np.random.default_rng(seed)
    kp = [np.concatenate([w.priv_k(e), w.k_new[e:e + 1]]) for e in range(w.n_events)]
    vp = [np.concatenate([w.priv_v(e), w.v_new[e:e + 1]]) for e in range(w.n_events)]
    lens = (w.event_len + 1).astype(np.int32)
    off = np.zeros(w.n_events + 1, np.int64)
    off[1:] = np.cumsum(lens)

    def draw(shape):
        return synth.f32_to_bf16_bits(rng.standard_normal(shape).astype(np.float32))

    return dataclasses.replace(w, event_len=lens, priv_off=off, k_priv=np.concatenate(kp),
                               v_priv=np.concatenate(vp), q=draw(w.q.shape), k_new=draw(w.k_new.shape),
                               v_new=draw(w.v_new.shape), page_table=pt, free_pages=free)


@pytest.mark.gpu
@pytest.mark.parametrize("flags", [0, B.FLAG_PREFIX_DUAL])
def test_host_only_plans_run_two_steps_against_the_oracle(padlib, flags):
    """A caller with no device scratch runs two consecutive steps with pad_kv_append +
    pad_event_decode_attn_static on plans built without a workspace: branches on page
    boundaries open pages in the first step and others in the second; the outputs match the
    fp64 oracle and the page table the simulated bookkeeping, after both steps."""
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import oracle
    from paper_2607_02963_gb300.device import bits_to_bf16
    rng = np.random.default_rng(3)
    w = synth.make_workload("host_only", 3, 28, 4, 128, [1500, 700], [3, 2], [0, 15, 16, 31, 47], rng=rng)
    db = DeviceBatch(w)
    for step in range(2):
        if step:
            w = _next_step(w, 40 + step)
            db.q.copy_(bits_to_bf16(w.q, db.device))
            db.k_new.copy_(bits_to_bf16(w.k_new, db.device))
            db.v_new.copy_(bits_to_bf16(w.v_new, db.device))
        prob = B.make_problem(w.h_q, w.h_kv, w.head_dim, w.page_size, w.scale, flags=flags)
        plan = B.pad_plan(prob, db.cache, w.prefix_len, w.event_video, w.event_len,
                          page_table=db.page_table, max_pages=w.max_pages, workspace=None,
                          prefix_offset=w.prefix_offset)
        B.pad_kv_append(plan, db.k_new, db.v_new, db.k_pool, db.v_pool)
        o = torch.full_like(db.out, float("nan"))
        lse = torch.full_like(db.lse, float("nan"))
        B.pad_event_decode_attn_static(plan, db.q, db.k_prefix, db.v_prefix, db.k_pool, db.v_pool, o, lse)
        torch.cuda.synchronize()
        B.pad_device_status(plan)
        st, pt, _, _ = oracle.simulate_append(w.page_table, w.free_pages, w.event_len, w.page_size)
        assert st == oracle.OK
        assert np.array_equal(db.page_table.cpu().numpy(), pt), f"page table after step {step}"
        ref_o, ref_l = oracle.decode_step(w)
        _compare(o, lse, torch.from_numpy(ref_o), torch.from_numpy(ref_l))


@pytest.mark.gpu
def test_static_path_reports_device_errors(padlib):
    """An out-of-pool page id met by the kernels on the static path is reported by
    pad_device_status for that plan (the status word lives in the static array), and a
    clean step afterwards on the same array runs and reports nothing."""
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    w = synth.make_workload("static_bad", 7, 28, 4, 128, [200], [2], [5, 3])
    db = DeviceBatch(w)
    good = int(db.page_table[1, 0])
    db.page_table[1, 0] = w.n_pages + 5
    plan = B.pad_plan(db.problem, db.cache, w.prefix_len, w.event_video, w.event_len,
                      page_table=db.page_table, max_pages=w.max_pages, workspace=None,
                      prefix_offset=w.prefix_offset)
    B.pad_kv_append(plan, db.k_new, db.v_new, db.k_pool, db.v_pool)
    B.pad_event_decode_attn_static(plan, db.q, db.k_prefix, db.v_prefix, db.k_pool, db.v_pool,
                                   db.out, db.lse)
    with pytest.raises(B.PadError) as ei:
        B.pad_device_status(plan)
    assert ei.value.status == 7
    plan.release_new_pages(db.cache)
    db.page_table[1, 0] = good
    plan2 = B.pad_plan(db.problem, db.cache, w.prefix_len, w.event_video, w.event_len,
                       page_table=db.page_table, max_pages=w.max_pages, workspace=None,
                       prefix_offset=w.prefix_offset)
    B.pad_kv_append(plan2, db.k_new, db.v_new, db.k_pool, db.v_pool)
    B.pad_event_decode_attn_static(plan2, db.q, db.k_prefix, db.v_prefix, db.k_pool, db.v_pool,
                                   db.out, db.lse)
    torch.cuda.synchronize()
    B.pad_device_status(plan2)
    import oracle
    ref_o, ref_l = oracle.decode_step(w)
    _compare(db.out, db.lse, torch.from_numpy(ref_o), torch.from_numpy(ref_l))


@pytest.mark.gpu
def test_plan_just_under_the_static_limit(padlib):
    """A plan whose scratch is just under the array's 16 MiB runs on the static path and
    matches the workspace path of the same step."""
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    # videos of E events x 7 q-heads per kv-head with short prefixes: the partial states grow
    # with the videos, the events and the splits the planner gives them; take the largest
    # scratch that still fits
    prob = B.make_problem(28, 4, 128, num_sms=152)
    best = None
    for nv in range(1, 24):
        for E in (64, 56, 48, 40, 32):
            ev = np.repeat(np.arange(nv, dtype=np.int32), E)
            ws = B.pad_workspace_size(prob, np.full(nv, 300, np.int32), ev)
            if ws <= 16 << 20 and (best is None or ws > best[2]):
                best = (nv, E, ws)
    assert best is not None and best[2] > 15 << 20
    nv, E = best[0], best[1]
    rng = np.random.default_rng(11)
    w = synth.make_workload("near_limit", 11, 28, 4, 128, [300] * nv, [E] * nv,
                            rng.integers(0, 40, size=E * nv), rng=rng)
    db = DeviceBatch(w, num_sms=152)
    plan = db.run_step()
    torch.cuda.synchronize()
    B.pad_device_status(plan)
    assert plan.info()["workspace_bytes"] == best[2]
    ref_o, ref_l = db.out.clone(), db.lse.clone()
    db.release_new_pages(plan)
    hplan = B.pad_plan(db.problem, db.cache, w.prefix_len, w.event_video, w.event_len,
                       page_table=db.page_table, max_pages=w.max_pages, workspace=None,
                       prefix_offset=w.prefix_offset)
    o = torch.full_like(db.out, float("nan"))
    lse = torch.full_like(db.lse, float("nan"))
    B.pad_event_decode_attn_static(hplan, db.q, db.k_prefix, db.v_prefix, db.k_pool, db.v_pool, o, lse)
    torch.cuda.synchronize()
    B.pad_device_status(hplan)
    _compare(o, lse, ref_o, ref_l)
