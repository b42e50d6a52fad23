"""Host logic of the C ABI (no GPU): page bookkeeping of pad_plan against the oracle's
simulation (bit-exact), the split-KV work list, and argument validation."""
import json
import os

import numpy as np
import pytest

import oracle
from paper_2607_02963_gb300 import binding as B
from paper_2607_02963_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _dry_plan(prob, cache, w_like):
    return B.pad_plan(prob, cache, w_like["prefix_len"], w_like["event_video"], w_like["event_len"],
                      page_table=None, max_pages=w_like["max_pages"], workspace=None)


def test_hand_worked_page_append(padlib):
    g = json.load(open(os.path.join(GOLDEN, "hand_page_append.json")))
    pt = np.array(g["page_table"], dtype=np.int32)
    n_pages = 10
    used = pt[pt >= 0]
    cache = B.CacheState(n_pages, used_pages=used)
    assert sorted(cache.free_pages().tolist()) == g["free_pages"]
    prob = B.make_problem(4, 2, 64, page_size=g["page_size"], num_sms=8)
    E = len(g["event_len"])
    plan = _dry_plan(prob, cache, dict(prefix_len=[8], event_video=[0] * E,
                                       event_len=g["event_len"], max_pages=pt.shape[1]))
    new = plan.new_pages()
    expect = np.array(g["expect_page_table"])
    for e, L in enumerate(g["event_len"]):
        if L % g["page_size"] == 0:
            assert new[e] == expect[e, L // g["page_size"]]
        else:
            assert new[e] == -1
    assert cache.free_pages().tolist() == g["expect_free_pages"]
    # out of pages: nothing changes
    cache2 = B.CacheState(n_pages, used_pages=[p for p in range(n_pages) if p not in (0, 3)])
    before = cache2.export().copy()
    with pytest.raises(B.PadError) as ei:
        _dry_plan(prob, cache2, dict(prefix_len=[8], event_video=[0] * E, event_len=g["event_len"],
                                     max_pages=pt.shape[1]))
    assert ei.value.status == 3
    assert np.array_equal(cache2.export(), before)


@pytest.mark.parametrize("seed", range(8))
def test_page_allocation_matches_oracle_simulation(padlib, seed):
    w = synth.random_small(seed, max_events=9, max_len=70, max_prefix=300)
    cache = B.CacheState(w.n_pages, used_pages=w.page_table[w.page_table >= 0])
    prob = B.make_problem(w.h_q, w.h_kv, w.head_dim, w.page_size, num_sms=16)
    plan = _dry_plan(prob, cache, dict(prefix_len=w.prefix_len, event_video=w.event_video,
                                       event_len=w.event_len, max_pages=w.max_pages))
    st, pt, free, slots = oracle.simulate_append(w.page_table, w.free_pages, w.event_len, w.page_size)
    assert st == oracle.OK
    new = plan.new_pages()
    for e in range(w.n_events):
        L = int(w.event_len[e])
        if L % w.page_size == 0:
            assert new[e] == pt[e, L // w.page_size]
        else:
            assert new[e] == -1
    assert np.array_equal(cache.free_pages(), free)
    assert plan.info()["n_new_pages"] == int(np.sum(w.event_len % w.page_size == 0))


def test_split_work_list_covers_each_prefix_once(padlib):
    w = synth.ragged_serving.__wrapped__ if hasattr(synth.ragged_serving, "__wrapped__") else None
    rng = np.random.default_rng(0)
    P = rng.integers(1, 5000, size=7).astype(np.int32)
    Ev = rng.integers(0, 5, size=7)
    P[3] = 0
    ev_video = np.repeat(np.arange(7, dtype=np.int32), Ev)
    L = np.zeros(ev_video.size, dtype=np.int32) + 3
    cache = B.CacheState(64)
    prob = B.make_problem(28, 4, 128, num_sms=152)
    plan = B.pad_plan(prob, cache, P, ev_video, L, max_pages=2, workspace=None)
    info = plan.info()
    sl = info["split_len"]
    assert sl % 128 == 0
    expect_items = sum(4 * -(-int(P[b]) // sl) for b in range(7) if Ev[b] > 0 and P[b] > 0)
    assert info["n_work_items"] == expect_items
    expect_rows = sum(4 * -(-int(P[b]) // sl) * int(Ev[b]) * 7 for b in range(7) if P[b] > 0)
    assert info["partial_rows"] == expect_rows
    ws = B.pad_workspace_size(prob, P, ev_video)
    assert ws == info["workspace_bytes"] and ws % 256 == 0


def test_workload_sizes_and_kernel_choice(padlib):
    prob = B.make_problem(28, 4, 128, num_sms=148)
    cache = B.CacheState(1000)
    # head_dim 128: tensor-core path; 32 events -> R = 224 rows = two 128-row groups per
    # item, and items x groups fill one wave of SMs without exceeding it
    plan = B.pad_plan(prob, cache, [32768], [0] * 32, [1] * 32, max_pages=4, workspace=None)
    info = plan.info()
    assert info["prefix_kernel"] == B.FLAG_PREFIX_TC
    assert 120 <= 2 * info["n_work_items"] <= 148
    plan = B.pad_plan(prob, cache, [16384], [0], [1], max_pages=4, workspace=None)
    assert plan.info()["prefix_kernel"] == B.FLAG_PREFIX_TC
    assert plan.info()["n_work_items"] <= 148
    # forced: the dual kernel, one 256-row CTA per item
    prob_d = B.make_problem(28, 4, 128, num_sms=148, flags=B.FLAG_PREFIX_DUAL)
    info = B.pad_plan(prob_d, cache, [32768], [0] * 32, [1] * 32, max_pages=4, workspace=None).info()
    assert info["prefix_kernel"] == B.FLAG_PREFIX_DUAL
    assert 130 <= info["n_work_items"] <= 148
    # the fused tail asks for the single-group kernel
    prob_f = B.make_problem(28, 4, 128, num_sms=148, flags=B.FLAG_FUSED_MERGE)
    info = B.pad_plan(prob_f, cache, [32768], [0] * 32, [1] * 32, max_pages=4, workspace=None).info()
    assert info["prefix_kernel"] == B.FLAG_PREFIX_TC
    # head_dim 64: warp-level paths, warp-shuffle for <= 8 rows
    prob64 = B.make_problem(16, 4, 64, num_sms=148)
    plan = B.pad_plan(prob64, cache, [4096], [0, 0], [1, 1], max_pages=4, workspace=None)
    assert plan.info()["prefix_kernel"] == B.FLAG_PREFIX_SIMT
    plan = B.pad_plan(prob64, cache, [4096], [0, 0, 0], [1, 1, 1], max_pages=4, workspace=None)
    assert plan.info()["prefix_kernel"] == B.FLAG_PREFIX_MMA


@pytest.mark.parametrize("flags,rows_per_cta", [(0, 128), (B.FLAG_PREFIX_DUAL, 256)])
def test_tc_split_fits_one_wave(padlib, flags, rows_per_cta):
    rng = np.random.default_rng(5)
    for trial in range(50):
        B_ = int(rng.integers(1, 17))
        P = rng.integers(1, 40000, size=B_).astype(np.int32)
        Ev = rng.integers(1, 40, size=B_)
        ev_video = np.repeat(np.arange(B_, dtype=np.int32), Ev)
        L = np.zeros(ev_video.size, dtype=np.int32)
        sms = int(rng.integers(8, 160))
        prob = B.make_problem(28, 4, 128, num_sms=sms, flags=flags)
        plan = B.pad_plan(prob, B.CacheState(4096), P, ev_video, L, max_pages=2, workspace=None)
        info = plan.info()
        sl = info["split_len"]
        assert sl % 128 == 0
        # each work item gets the row groups its own video needs (a CTA list, not a dense
        # grid of the largest count): one wave unless a single split per (video, kv-head)
        # is already too many
        groups = [-(-int(Ev[b]) * 7 // rows_per_cta) for b in range(B_)]
        if B_ == 1:
            ctas = sum(4 * -(-int(P[b]) // sl) * groups[b] for b in range(B_))
            items = sum(4 * -(-int(P[b]) // sl) for b in range(B_))
            assert info["n_work_items"] == items
            assert info["prefix_ctas"] == ctas
            if sl < int(P.max()):
                assert ctas <= sms
        else:
            # a batch of videos: per-video splits, a grid of at most three waves unless one
            # split per (video, kv-head, row group) is already more
            base = sum(4 * g for g in groups)
            assert base <= info["prefix_ctas"] <= max(base, 3 * sms)
            assert info["max_split_tiles"] == sl // 128
            assert 4 * B_ <= info["n_work_items"] <= info["prefix_ctas"]


def _split_of(P, E, sms=152, flags=0):
    prob = B.make_problem(28, 4, 128, num_sms=sms, flags=flags)
    ev = np.zeros(E, np.int32)
    plan = B.pad_plan(prob, B.CacheState(4096), np.array([P], np.int32), ev, np.zeros(E, np.int32),
                      max_pages=2, workspace=None)
    return plan.info()["split_len"]


def test_tc_split_leaves_sms_for_the_branch_tasks(padlib):
    """The planner takes a split up to two tiles longer than the one-wave minimum when that
    leaves an SM for every (event, kv-head) branch task and the extra tiles cost less than
    running the tasks' pre-wait part after the prefix pass (0.85 us per tile, 2 us)."""
    # 16384-token prefix, 4 kv-heads, one row group: 128 one-wave CTAs of 4 tiles
    assert _split_of(16384, 4) == 512        # 16 tasks fit the 24 free SMs already
    assert _split_of(16384, 8) == 640        # 32 tasks: 104 CTAs of 5 tiles leave 48 SMs
    assert _split_of(16384, 16) == 768       # 64 tasks: 88 CTAs of 6 tiles leave 64 SMs
    assert _split_of(8192, 8) == 384         # gqa_8k: 88 CTAs of 3 tiles
    # 128 tasks never fit beside a one-wave grid: the minimum split stays
    assert _split_of(32768, 32) == 1792
    # the fused tail plans its own grid
    assert _split_of(16384, 8, flags=B.FLAG_FUSED_MERGE) == 512
    # every candidate stays within one wave
    for E in (1, 3, 8, 12, 20):
        sl = _split_of(16384, E, sms=100)
        groups = -(-E * 7 // 128)
        assert 4 * -(-16384 // sl) * groups <= 100


def _info_of(P, E, sms=152, flags=0):
    prob = B.make_problem(28, 4, 128, num_sms=sms, flags=flags)
    ev = np.zeros(E, np.int32)
    plan = B.pad_plan(prob, B.CacheState(4096), np.array([P], np.int32), ev, np.zeros(E, np.int32),
                      max_pages=2, workspace=None)
    return plan.info()


def test_branch_tasks_wait_first_only_when_no_slot_is_left_beside_the_prefix_grid(padlib):
    """merge_first: the branch tasks wait for the prefix pass before their branch pass when
    some (event, kv-head) task cannot get one of the two slots of each SM that the one-wave
    tensor-core grid leaves free; otherwise they run their branch pass beside it."""
    # 32 events x 4 kv-heads = 128 tasks beside a 152-CTA grid: no free SM
    info = _info_of(32768, 32)
    assert info["prefix_ctas"] == 152 and info["merge_first"] == 1
    # 64 tasks beside 88 CTAs: 128 free slots
    info = _info_of(16384, 16)
    assert info["prefix_ctas"] == 88 and info["merge_first"] == 0
    # one event: 4 tasks, 24 free SMs
    assert _info_of(16384, 1)["merge_first"] == 0
    # a smaller GPU: the split grows to keep one wave, still with no SM free
    assert _info_of(32768, 32, sms=64)["merge_first"] == 1
    # a second wave (4 row groups x 4 kv-heads on 8 SMs) keeps the branch pass before the wait
    info = _info_of(16384, 64, sms=8)
    assert info["prefix_ctas"] > 8 and info["merge_first"] == 0
    # the fused tail runs its tasks in the prefix kernel
    assert _info_of(16384, 8, flags=B.FLAG_FUSED_MERGE)["merge_first"] == 0
    # every rule in one place: tasks > 2 x free SMs of a one-wave grid
    for P, E in ((16384, 32), (16384, 64), (8192, 8), (65536, 4), (4096, 40)):
        info = _info_of(P, E)
        free = 152 - info["prefix_ctas"]
        want = int(info["prefix_ctas"] <= 152 and E * 4 > 2 * free)
        assert info["merge_first"] == want, (P, E, info)


def test_batch_of_videos_takes_balanced_splits_over_several_waves(padlib):
    """16 videos of 4k-16k prefix tokens (the ragged serving batch): one split length sized
    to one wave leaves CTAs of 82 tiles beside CTAs of 32; per-video splits over two waves,
    longest first, bring the longest CTA to 32 tiles."""
    w = synth.ragged_serving()
    prob = B.make_problem(w.h_q, w.h_kv, w.head_dim, w.page_size, num_sms=152)
    cache = B.CacheState(w.n_pages, used_pages=w.page_table[w.page_table >= 0])
    plan = B.pad_plan(prob, cache, w.prefix_len, w.event_video, w.event_len, max_pages=w.max_pages,
                      workspace=None)
    info = plan.info()
    plan.release_new_pages(cache)
    assert 152 < info["prefix_ctas"] <= 2 * 152
    assert info["max_split_tiles"] <= 32
    # the same batch forced to one split length per video when there is a single video
    w1 = synth.make_workload("one", 3, 28, 4, 128, [16000], [20], [5] * 20, rng=np.random.default_rng(3))
    p1 = B.pad_plan(prob, B.CacheState(w1.n_pages, used_pages=w1.page_table[w1.page_table >= 0]),
                    w1.prefix_len, w1.event_video, w1.event_len, max_pages=w1.max_pages, workspace=None)
    assert p1.info()["prefix_ctas"] <= 152


@pytest.mark.parametrize("case,status", [
    (dict(event_video=[1, 0]), 1),                       # not sorted by video
    (dict(event_video=[0, 2]), 1),                       # video out of range
    (dict(event_len=[-1, 0]), 1),                        # negative length
    (dict(event_len=[64, 0]), 1),                        # page index beyond max_pages
    (dict(head_dim=96), 2),                              # unsupported head_dim
    (dict(h_q=6, h_kv=4), 1),                            # h_q not a multiple of h_kv
    (dict(page_size=12), 2),                             # unsupported page size
    (dict(h_q=34, h_kv=2), 2),                           # group 17 > 16
    (dict(prefix_len=[-3, 4]), 1),                       # negative prefix
])
def test_invalid_arguments_change_nothing(padlib, case, status):
    args = dict(event_video=[0, 1], event_len=[3, 0], prefix_len=[100, 50], h_q=8, h_kv=2,
                head_dim=64, page_size=16, max_pages=4)
    args.update(case)
    prob = B.make_problem(args["h_q"], args["h_kv"], args["head_dim"], args["page_size"])
    cache = B.CacheState(16)
    before = cache.export().copy()
    with pytest.raises(B.PadError) as ei:
        B.pad_plan(prob, cache, args["prefix_len"], args["event_video"], args["event_len"],
                   max_pages=args["max_pages"], workspace=None)
    assert ei.value.status == status
    assert np.array_equal(cache.export(), before)


def test_empty_step(padlib):
    prob = B.make_problem(8, 2, 64)
    cache = B.CacheState(4)
    plan = B.pad_plan(prob, cache, [10], [], [], max_pages=1, workspace=None)
    info = plan.info()
    assert info["n_events"] == 0 and info["n_work_items"] == 0 and info["n_new_pages"] == 0
    plan = B.pad_plan(prob, cache, [], [], [], max_pages=1, workspace=None)
    assert plan.info()["n_work_items"] == 0


def test_cache_state_checkpoint_and_errors(padlib):
    c = B.CacheState(10, used_pages=[1, 4, 5])
    assert c.free_count == 7
    snap = c.export()
    with pytest.raises(B.PadError):
        c.mark_used([4])          # already used
    with pytest.raises(B.PadError):
        c.release([2])            # already free
    with pytest.raises(B.PadError):
        c.mark_used([10])         # out of range
    with pytest.raises(B.PadError):
        c.mark_used([2, 2])       # listed twice
    assert np.array_equal(c.export(), snap)
    c.release([1, 4])
    assert c.free_count == 9
    c2 = B.CacheState(10)
    c2.import_(snap)
    assert c2.free_count == 7 and np.array_equal(c2.export(), snap)
    with pytest.raises(B.PadError):
        c2.import_(np.zeros(9, dtype=np.uint8))


def test_launch_calls_reject_plans_without_workspace(padlib):
    prob = B.make_problem(8, 2, 64)
    cache = B.CacheState(4)
    plan = B.pad_plan(prob, cache, [10], [0], [0], max_pages=1, workspace=None)
    with pytest.raises(B.PadError) as ei:
        B.lib().pad_kv_append(plan.handle, None, None, None, None, None) and None
        B._check(B.lib().pad_kv_append(plan.handle, None, None, None, None, None))
    assert ei.value.status == 1


def test_release_new_pages_returns_exactly_the_plans_pages(padlib):
    """pad_plan_release_new_pages frees the pages the plan took and nothing else; releasing
    twice is an error that changes nothing."""
    cache = B.CacheState(40, used_pages=[0, 1, 2, 5])
    prob = B.make_problem(4, 1, 64, page_size=16)
    lens = np.array([16, 3, 32, 0], dtype=np.int32)  # three page starts
    plan = B.pad_plan(prob, cache, [100], [0, 0, 0, 0], lens, max_pages=4, workspace=None)
    new = plan.new_pages()
    assert sorted(new[new >= 0].tolist()) == [3, 4, 6]
    free_before = cache.free_count
    plan.release_new_pages(cache)
    assert cache.free_count == free_before + 3
    assert sorted(cache.free_pages().tolist()) == [p for p in range(40) if p not in (0, 1, 2, 5)]
    with pytest.raises(B.PadError) as ei:
        plan.release_new_pages(cache)
    assert ei.value.status == 1
    assert cache.free_count == free_before + 3


def test_fused_tail_decision(padlib):
    """The tensor-core plan runs a4 + a5 inside the prefix kernel exactly when every
    (event, kv-head) task can have a prefix CTA of its own and the prefix grid fits one
    CTA per SM (the tail waits on other CTAs' splits, so the grid must be resident at
    once), and only when PAD_FLAG_FUSED_MERGE asks for it."""
    rng = np.random.default_rng(17)
    seen = set()
    for trial in range(80):
        B_ = int(rng.integers(1, 6))
        P = rng.integers(0, 30000, size=B_).astype(np.int32)
        Ev = rng.integers(1, 24, size=B_)
        ev_video = np.repeat(np.arange(B_, dtype=np.int32), Ev)
        L = np.zeros(ev_video.size, dtype=np.int32)
        sms = int(rng.integers(8, 160))
        for flags in (0, B.FLAG_FUSED_MERGE, B.FLAG_PREFIX_TC | B.FLAG_FUSED_MERGE):
            prob = B.make_problem(28, 4, 128, num_sms=sms, flags=flags)
            info = B.pad_plan(prob, B.CacheState(4096), P, ev_video, L, max_pages=2, workspace=None).info()
            sl = info["split_len"]
            groups = max(-(-int(Ev[b]) * 7 // 128) for b in range(B_))
            valid = sum(4 * (-(-int(P[b]) // sl)) * (-(-int(Ev[b]) * 7 // 128)) for b in range(B_))
            want = (bool(flags & B.FLAG_FUSED_MERGE) and info["n_work_items"] > 0 and info["n_work_items"] * groups <= sms
                    and int(Ev.sum()) * 4 <= valid)
            assert info["fused_tail"] == int(want), (trial, flags)
            seen.add(want)
    assert seen == {True, False}
    # the 64-dim problems never take the tensor-core path, hence never the fused tail
    prob = B.make_problem(8, 2, 64, num_sms=152, flags=B.FLAG_FUSED_MERGE)
    info = B.pad_plan(prob, B.CacheState(64), np.array([5000], np.int32), np.zeros(2, np.int32),
                      np.zeros(2, np.int32), max_pages=2, workspace=None).info()
    assert info["fused_tail"] == 0


def test_set_rope_validates_positions_and_table(padlib):
    import torch
    prob = B.make_problem(8, 2, 128, num_sms=152)
    cache = B.CacheState(64)
    plan = B.pad_plan(prob, cache, np.array([500], np.int32), np.zeros(3, np.int32),
                      np.array([0, 3, 16], np.int32), max_pages=4, workspace=None)
    table = torch.zeros((100, 128), dtype=torch.float32)
    plan.set_rope(np.array([0, 50, 99], np.int32), table)
    for bad in ([0, 50, 100], [-1, 0, 0]):
        with pytest.raises(B.PadError) as ei:
            plan.set_rope(np.array(bad, np.int32), table)
        assert ei.value.status == 1
    with pytest.raises(B.PadError) as ei:
        B._check(B.lib().pad_plan_set_rope(plan.handle, np.zeros(3, np.int32).ctypes.data_as(B._I32P), None, 100))
    assert ei.value.status == 1


def test_set_g_visibility_validates(padlib):
    prob = B.make_problem(8, 2, 128, num_sms=152)
    plan = B.pad_plan(prob, B.CacheState(64), np.array([50, 10], np.int32), np.array([0, 0, 1], np.int32),
                      np.array([0, 3, 16], np.int32), max_pages=4, workspace=None)
    plan.set_g_visibility(B.G_SELF, [4, 9], [0, 3, 8])
    plan.set_g_visibility(B.G_ALL)
    for K, gi in (([50, 0], [0, 0, 0]),      # K + 1 > prefix
                  ([4, 2], [0, 4, 1]),       # index >= K
                  ([4, 0], [0, 1, 1]),       # K = 0 needs index 0
                  ([-1, 2], [0, 0, 0])):
        with pytest.raises(B.PadError) as ei:
            plan.set_g_visibility(B.G_SELF, K, gi)
        assert ei.value.status == 1
    with pytest.raises(B.PadError):
        plan.set_g_visibility(7)


def test_set_branch_visibility_validates(padlib):
    prob = B.make_problem(8, 2, 128, num_sms=152)
    plan = B.pad_plan(prob, B.CacheState(64), np.array([50], np.int32), np.zeros(2, np.int32),
                      np.array([3, 16], np.int32), max_pages=4, workspace=None)
    plan.set_branch_visibility(B.BRANCH_CAUSAL)
    plan.set_branch_visibility(B.BRANCH_OWN)
    with pytest.raises(B.PadError) as ei:
        plan.set_branch_visibility(2)
    assert ei.value.status == 1


def test_step_executor_validates_and_returns_pages_of_a_failed_run(padlib):
    """pad_step_create checks its arguments; a run whose launch fails (no device here, or a
    refused launch) hands the pages its plan took back to the cache."""
    import ctypes
    prob = B.make_problem(8, 2, 128, num_sms=152)
    cache = B.CacheState(64)
    pl = np.array([500], np.int32)
    ev = np.zeros(3, np.int32)
    el = np.array([0, 16, 5], np.int32)  # two events start pages
    h = ctypes.c_void_p()
    fake = 1 << 20  # 16-byte aligned addresses, never dereferenced by the host
    args = [ctypes.byref(prob), cache.handle, 1, pl.ctypes.data_as(B._I32P), None, 3, ev.ctypes.data_as(B._I32P),
            el.ctypes.data_as(B._I32P), fake, 4, fake, 1 << 24] + [fake] * 9 + [None]
    for bad_opts in (0x8, -1):
        with pytest.raises(B.PadError) as ei:
            B._check(B.lib().pad_step_create(*args, bad_opts, ctypes.byref(h)))
        assert ei.value.status == 1
    no_ws = list(args)
    no_ws[10] = None
    with pytest.raises(B.PadError) as ei:
        B._check(B.lib().pad_step_create(*no_ws, 0, ctypes.byref(h)))
    assert ei.value.status == 1
    B._check(B.lib().pad_step_create(*args, B.STEP_MAPPED_HOST_IO, ctypes.byref(h)))
    B.lib().pad_step_destroy(h)
    B._check(B.lib().pad_step_create(*args, 0, ctypes.byref(h)))
    try:
        import torch
        if not torch.cuda.is_available():
            # without a device the launch is refused before any kernel runs (with one, the
            # fake addresses above must never reach a kernel: this part is skipped)
            free0 = cache.free_count
            new = np.full(3, -7, np.int32)
            st = B.lib().pad_step_run(h, new.ctypes.data_as(B._I32P))
            assert st != 0
            assert cache.free_count == free0
    finally:
        B.lib().pad_step_destroy(h)


def test_attn_aggregate_workspace_and_argument_checks(padlib):
    """The aggregation's scratch is (n_segments + ceil(n_tokens / 256)) x (d_model + 1) fp32;
    a smaller one, a hidden size that is not a multiple of 8, a NULL tensor or a misaligned
    one are refused before anything is launched (no device is touched here)."""
    import ctypes
    L = B.lib()
    for T, S, d in ((32768, 128, 2048), (3400, 3, 520), (1, 1, 8), (256, 1, 64), (257, 1, 64)):
        assert L.pad_attn_aggregate_workspace_size(T, S, d) == (S + -(-T // 256)) * (d + 1) * 4
    assert L.pad_attn_aggregate_workspace_size(-1, 1, 8) == 0
    assert L.pad_attn_aggregate_workspace_size(10, 0, 8) == 0
    off = np.array([0, 100, 300], np.int32)
    a = 1 << 20  # 16-byte aligned addresses, never dereferenced: every call below fails its checks
    need = L.pad_attn_aggregate_workspace_size(300, 2, 64)

    def call(d=64, ws_bytes=need, x=a, ws=a, n_events=3):
        return L.pad_attn_aggregate(x, 300, d, a, off.ctypes.data_as(B._I32P), 2, a, n_events, a, ws, ws_bytes, a,
                                    None)
    assert call(ws_bytes=need - 4) == 4                      # PAD_ERR_WORKSPACE_TOO_SMALL
    assert call(d=60) == 2                                   # d_model not a multiple of 8
    assert call(ws=None) == 1                                # NULL scratch
    assert call(ws=a + 4) == 1                               # misaligned scratch
    assert call(x=a + 8) == 1                                # misaligned hidden states
    bad = np.array([0, 301, 300], np.int32)                  # offsets past n_tokens
    assert L.pad_attn_aggregate(a, 300, 64, a, bad.ctypes.data_as(B._I32P), 2, a, 3, a, a, need, a, None) == 1


def test_step_executor_setters_validate(padlib):
    """pad_step_set_*: a NULL executor, an unknown mode, and the arrays a mode needs."""
    import ctypes
    L = B.lib()
    assert L.pad_step_run(None, None) == 1
    assert L.pad_step_set_branch_visibility(None, B.BRANCH_CAUSAL) == 1
    prob = B.make_problem(8, 2, 128, num_sms=152)
    cache = B.CacheState(64)
    pl = np.array([500], np.int32)
    ev = np.zeros(2, np.int32)
    el = np.array([3, 7], np.int32)
    fake = 1 << 20  # never dereferenced: nothing below launches
    h = ctypes.c_void_p()
    B._check(L.pad_step_create(ctypes.byref(prob), cache.handle, 1, pl.ctypes.data_as(B._I32P), None, 2,
                               ev.ctypes.data_as(B._I32P), el.ctypes.data_as(B._I32P), fake, 4, fake, 1 << 24,
                               *([fake] * 9), None, 0, ctypes.byref(h)))
    try:
        assert L.pad_step_set_branch_visibility(h, 2) == 1
        assert L.pad_step_set_branch_visibility(h, B.BRANCH_CAUSAL) == 0
        assert L.pad_step_set_branch_visibility(h, B.BRANCH_OWN) == 0
        assert L.pad_step_set_g_visibility(h, 5, None, None) == 1
        assert L.pad_step_set_g_visibility(h, B.G_SELF, None, None) == 1   # K / G indices needed
        assert L.pad_step_set_g_visibility(h, B.G_ALL, None, None) == 0
        assert L.pad_step_set_rope(h, None, fake, 100) == 1                # positions needed
        assert L.pad_step_set_rope(h, None, fake + 4, 100) == 1            # misaligned table
        pos = np.zeros(2, np.int32)
        assert L.pad_step_set_rope(h, pos.ctypes.data_as(B._I32P), fake, 0) == 1
        assert L.pad_step_set_rope(h, pos.ctypes.data_as(B._I32P), fake, 100) == 0
        assert L.pad_step_set_rope(h, None, None, 0) == 0                  # off again
    finally:
        L.pad_step_destroy(h)
