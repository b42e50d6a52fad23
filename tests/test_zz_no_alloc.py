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
