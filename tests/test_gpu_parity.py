"""Parity of the CUDA path (through the C ABI) against the fp64 oracle.

Bar (from the problem statement): page-table and pool bookkeeping bit-exact;
outputs within max-abs <= 1e-2 and relative-L2 <= 2e-3 (bf16 in, fp32
accumulate); the natural-log LSE within 1e-3 absolute (a log of an fp32 sum of
positive terms: its error is the relative error of that sum, ~1e-6 here).
"""
import hashlib

import numpy as np
import pytest
import torch

import oracle
from paper_2607_02963_gb300 import binding as B
from paper_2607_02963_gb300 import synth
from paper_2607_02963_gb300.device import DeviceBatch

pytestmark = pytest.mark.gpu

MAX_ABS = 1e-2
REL_L2 = 2e-3
LSE_ABS = 1e-3


@pytest.fixture(scope="module", autouse=True)
def _cuda(padlib):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.init()


def check_outputs(got_o, got_lse, ref_o, ref_lse, what=""):
    got_o = np.asarray(got_o, dtype=np.float64)
    assert np.all(np.isfinite(got_o)), f"{what}: non-finite output"
    err = np.abs(got_o - ref_o)
    rel = np.linalg.norm(got_o - ref_o) / np.linalg.norm(ref_o)
    assert err.max() <= MAX_ABS, f"{what}: max-abs {err.max():.3e}"
    assert rel <= REL_L2, f"{what}: rel-L2 {rel:.3e}"
    if got_lse is not None:
        lerr = np.abs(np.asarray(got_lse, dtype=np.float64) - ref_lse).max()
        assert lerr <= LSE_ABS, f"{what}: lse max-abs {lerr:.3e}"
    return err.max(), rel


def check_bookkeeping(db, w, plan):
    st, pt, free, slots = oracle.simulate_append(w.page_table, w.free_pages, w.event_len, w.page_size)
    assert st == oracle.OK
    assert np.array_equal(db.page_table.cpu().numpy(), pt), "page table differs from the simulation"
    assert np.array_equal(db.cache.free_pages(), free), "free pages differ from the simulation"
    new = plan.new_pages()
    for e in range(w.n_events):
        L = int(w.event_len[e])
        assert new[e] == (slots[e, 0] if L % w.page_size == 0 else -1)
    # every branch token, read back through the device page table, bit-equal to its source
    pages, offs, ks, vs = [], [], [], []
    for e in range(w.n_events):
        L = int(w.event_len[e])
        for t in range(L + 1):
            pages.append(pt[e, t // w.page_size])
            offs.append(t % w.page_size)
        ks.append(w.priv_k(e))
        ks.append(w.k_new[e:e + 1])
        vs.append(w.priv_v(e))
        vs.append(w.v_new[e:e + 1])
    pg = torch.tensor(pages, device=db.device, dtype=torch.long)
    of = torch.tensor(offs, device=db.device, dtype=torch.long)
    gk = db.k_pool[pg, :, of, :].view(torch.int16).cpu().numpy().view(np.uint16)
    gv = db.v_pool[pg, :, of, :].view(torch.int16).cpu().numpy().view(np.uint16)
    assert np.array_equal(gk, np.concatenate(ks)), "K pool contents differ"
    assert np.array_equal(gv, np.concatenate(vs)), "V pool contents differ"


_ORACLE = {}


def oracle_step(w):
    """fp64 oracle of the whole step (every event, every head), kept per workload so that
    the kernels compared on one workload share one oracle run."""
    h = hashlib.sha1()
    for a in (w.prefix_len, w.prefix_offset, w.event_video, w.event_len, w.q, w.k_prefix, w.v_prefix,
              w.k_priv, w.v_priv, w.k_new, w.v_new):
        h.update(np.ascontiguousarray(a).tobytes())
    key = (h.hexdigest(), w.h_q, w.h_kv, w.head_dim, w.scale)
    if key not in _ORACLE:
        _ORACLE.clear()
        _ORACLE[key] = oracle.decode_step(w)
    return _ORACLE[key]


def run_full(w, flags=0, out_dtype=0, what="", one_call=False):
    db = DeviceBatch(w, flags=flags, out_dtype=out_dtype)
    plan = db.run_step(one_call=one_call)
    torch.cuda.synchronize()
    B.pad_device_status(plan)
    check_bookkeeping(db, w, plan)
    ref_o, ref_lse = oracle_step(w)
    got = db.out.float().cpu().numpy()
    check_outputs(got, db.lse.cpu().numpy(), ref_o, ref_lse, what or w.name)
    return db, plan


# ---------------------------------------------------------------------------
# The five workloads
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("flags", [0, B.FLAG_PREFIX_SIMT, B.FLAG_PREFIX_MMA])
def test_tiny_full(flags):
    run_full(synth.tiny(), flags=flags)


@pytest.mark.parametrize("flags", [0, B.FLAG_PREFIX_MMA, B.FLAG_PREFIX_DUAL])
def test_gqa_8k_full(flags):
    run_full(synth.gqa_8k(), flags=flags)


# The full-size workloads: every output row of every event against the oracle, in the
# launch configuration the bench times (default flags: the tensor-core kernel; the one-call
# step, pad_decode_step), through the two-call step, and on the dual tensor-core kernel.
# In the one-call step on the tensor-core kernel, long_32k and the E = 32, 64 sweep points
# leave no SM free beside the prefix grid, so their branch tasks wait for it first
# (merge_first); the others run their branch pass beside it.
_MERGE_FIRST = {"long_32k": 1, "ragged_serving": 0, 1: 0, 2: 0, 4: 0, 8: 0, 16: 0, 32: 1, 64: 1}


def _check_merge_first(plan, key, flags):
    assert plan.info()["merge_first"] == (_MERGE_FIRST[key] if flags == 0 else 0)


@pytest.mark.parametrize("one_call", [True, False])
@pytest.mark.parametrize("flags", [0, B.FLAG_PREFIX_DUAL])
def test_long_32k_full(flags, one_call):
    _, plan = run_full(synth.long_32k(), flags=flags, one_call=one_call)
    _check_merge_first(plan, "long_32k", flags)


@pytest.mark.parametrize("one_call", [True, False])
@pytest.mark.parametrize("flags", [0, B.FLAG_PREFIX_DUAL])
def test_ragged_serving_full(flags, one_call):
    _, plan = run_full(synth.ragged_serving(), flags=flags, one_call=one_call)
    _check_merge_first(plan, "ragged_serving", flags)


# (E outermost, so that the cases of one workload share its oracle run)
@pytest.mark.parametrize("flags", [0, B.FLAG_PREFIX_DUAL])
@pytest.mark.parametrize("one_call", [True, False])
@pytest.mark.parametrize("E", synth.SWEEP_E)
def test_event_sweep_full(E, flags, one_call):
    _, plan = run_full(synth.event_sweep(E), flags=flags, one_call=one_call)
    _check_merge_first(plan, E, flags)


# ---------------------------------------------------------------------------
# Small random shapes (several tiles and a ragged tail), both prefix kernels
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("seed", range(6))
def test_random_small_mma(seed):
    run_full(synth.random_small(seed, h_q=8, h_kv=2, max_prefix=900, max_events=7),
             flags=B.FLAG_PREFIX_MMA)


@pytest.mark.parametrize("seed", range(6))
def test_random_small_tc(seed):
    run_full(synth.random_small(seed, h_q=8, h_kv=2, max_prefix=900, max_events=7),
             flags=B.FLAG_PREFIX_TC)


@pytest.mark.parametrize("seed", range(6))
def test_random_small_dual_tile_parity(seed):
    """<= 128 rows per item: the two softmax groups take alternate tiles of the same rows and
    their states are merged (odd and even tile counts, one-tile splits)."""
    run_full(synth.random_small(seed, h_q=8, h_kv=2, max_prefix=900, max_events=7),
             flags=B.FLAG_PREFIX_DUAL)


@pytest.mark.parametrize("E,prefix", [(19, 1000), (32, 130), (36, 100), (37, 1000), (64, 700), (40, 3000)])
def test_dual_row_groups(E, prefix):
    """> 128 rows per item (G = 7): two row groups share each tile (19 events: the second
    group holds 5 rows; 36: 252 rows); more than 256 rows take a second CTA (37 events: 256
    + 3 rows; 64: 256 + 192; 40: 256 + 24), whose last group may again fall back to tile
    parities; one- and two-tile splits and a ragged last tile."""
    lens = [(29 * i + 3) % 97 for i in range(E)]
    run_full(_w([prefix], [E], lens, seed=90 + E), flags=B.FLAG_PREFIX_DUAL, what=f"dual E {E} prefix {prefix}")


@pytest.mark.parametrize("seed", range(6))
def test_random_small_simt(seed):
    run_full(synth.random_small(seed, h_q=8, h_kv=2, max_prefix=900, max_events=4),
             flags=B.FLAG_PREFIX_SIMT)


@pytest.mark.parametrize("seed", range(3))
def test_random_small_head_dim_64(seed):
    w = synth.random_small(50 + seed, h_q=16, h_kv=4, head_dim=64, max_prefix=600, max_events=4)
    run_full(w, flags=B.FLAG_PREFIX_MMA)
    run_full(w, flags=B.FLAG_PREFIX_SIMT)


@pytest.mark.parametrize("flags", [B.FLAG_PREFIX_MMA, B.FLAG_PREFIX_TC, B.FLAG_PREFIX_DUAL])
def test_large_group_and_outlier_channels(flags):
    w = synth.random_small(60, h_q=32, h_kv=2, max_prefix=700, max_events=3, k_scale_sigma=0.5)
    run_full(w, flags=flags)


# ---------------------------------------------------------------------------
# Edge cases
# ---------------------------------------------------------------------------

def _w(prefix, epv, lens, seed=7, h_q=28, h_kv=4, D=128, sigma=None, page_size=16):
    rng = np.random.default_rng(seed)
    return synth.make_workload("edge", seed, h_q, h_kv, D, prefix, epv, lens, rng=rng,
                               k_scale_sigma=sigma, page_size=page_size)


@pytest.mark.parametrize("flags", [B.FLAG_PREFIX_TC, B.FLAG_PREFIX_DUAL])
@pytest.mark.parametrize("ps", [4, 8, 32, 64])
def test_page_sizes_many_events(ps, flags):
    """40 events of 7 rows (280 rows: three 128-row groups, two events straddling group
    boundaries) with branch lengths on and around page boundaries, for page sizes other
    than 16, over pools whose unwritten slots hold NaN."""
    lens = [(37 * i) % 131 for i in range(36)] + [ps, ps - 1, 2 * ps + 1, 0]
    run_full(_w([3000], [40], lens, seed=41 + ps, page_size=ps), flags=flags, what=f"ps {ps}")


@pytest.mark.parametrize("flags", [B.FLAG_PREFIX_SIMT, B.FLAG_PREFIX_MMA, B.FLAG_PREFIX_TC, B.FLAG_PREFIX_DUAL])
def test_single_event_empty_branch(flags):
    run_full(_w([300], [1], [0]), flags=flags)          # query sees the prefix and itself


@pytest.mark.parametrize("lens", [[16, 32, 0, 15, 17], [1, 31, 48, 63, 64]])
def test_page_boundaries(lens):
    run_full(_w([257], [len(lens)], lens))


@pytest.mark.parametrize("flags", [B.FLAG_PREFIX_MMA, B.FLAG_PREFIX_TC, B.FLAG_PREFIX_DUAL])
def test_prefix_not_multiple_of_tile_and_tiny_prefix(flags):
    run_full(_w([1, 129, 65], [2, 3, 2], [3, 0, 9, 16, 2, 5, 7]), flags=flags)


@pytest.mark.parametrize("flags", [B.FLAG_PREFIX_MMA, B.FLAG_PREFIX_TC, B.FLAG_PREFIX_DUAL])
def test_video_with_empty_prefix_and_video_without_events(flags):
    run_full(_w([0, 500, 200], [2, 0, 3], [4, 1, 0, 16, 2]), flags=flags)


@pytest.mark.parametrize("flags", [B.FLAG_PREFIX_MMA, B.FLAG_PREFIX_TC, B.FLAG_PREFIX_DUAL])
def test_sixty_four_events(flags):
    run_full(_w([700], [64], list(np.arange(64) % 40)), flags=flags)


@pytest.mark.parametrize("flags", [B.FLAG_PREFIX_TC, B.FLAG_PREFIX_DUAL])
def test_long_split_many_tiles_tc(flags):
    """Few SMs -> long splits: many tiles per CTA (the stage rings wrap several times, the S
    buffers alternate, lazy rescaling meets growing maxima)."""
    w = _w([5000, 3001], [5, 9], list(range(0, 70, 5)), sigma=0.5)
    db = DeviceBatch(w, flags=flags, num_sms=4)
    plan = db.run_step()
    torch.cuda.synchronize()
    B.pad_device_status(plan)
    assert plan.info()["split_len"] >= 2048
    ref_o, ref_lse = oracle.decode_step(w)
    check_outputs(db.out.cpu().numpy(), db.lse.cpu().numpy(), ref_o, ref_lse, "long splits")


def test_bf16_output():
    """bf16 output = round-to-nearest-even of the fp32 output of the same plan (bit-exact);
    against the oracle the bound grows by the rounding itself: |RNE(x) - x| <= 2^-9 |x|,
    so rel-L2 <= 2e-3 + 2^-9."""
    w = synth.random_small(3, h_q=8, h_kv=2, max_prefix=900, max_events=6)
    db32 = DeviceBatch(w, flags=B.FLAG_PREFIX_MMA, out_dtype=0)
    db32.run_step()
    db16 = DeviceBatch(w, flags=B.FLAG_PREFIX_MMA, out_dtype=1)
    plan = db16.run_step()
    torch.cuda.synchronize()
    B.pad_device_status(plan)
    assert db16.out.dtype == torch.bfloat16
    assert torch.equal(db16.out, db32.out.to(torch.bfloat16))
    ref_o, _ = oracle.decode_step(w)
    got = db16.out.double().cpu().numpy()
    assert np.abs(got - ref_o).max() <= MAX_ABS
    assert np.linalg.norm(got - ref_o) / np.linalg.norm(ref_o) <= REL_L2 + 2.0 ** -9


def test_empty_step_launches_nothing():
    w = _w([100], [1], [3])
    db = DeviceBatch(w)
    plan = B.pad_plan(db.problem, db.cache, w.prefix_len, w.event_video[:0], w.event_len[:0],
                      page_table=db.page_table, max_pages=w.max_pages, workspace=db.workspace)
    B.pad_kv_append(plan, db.k_new, db.v_new, db.k_pool, db.v_pool)
    B.pad_event_decode_attn(plan, db.q, db.k_prefix, db.v_prefix, db.k_pool, db.v_pool, db.out)
    torch.cuda.synchronize()


def test_repeated_steps_are_deterministic():
    w = synth.random_small(11, h_q=8, h_kv=2, max_prefix=900, max_events=6)
    db = DeviceBatch(w)
    db.run_step()
    o1 = db.out.clone()
    db.release_new_pages()
    db.run_step()
    torch.cuda.synchronize()
    assert torch.equal(o1, db.out)


@pytest.mark.parametrize("D,h_q", [(64, 4), (128, 8)])
def test_large_batch_reads_descriptors_from_host_image(D, h_q):
    """A batch whose descriptors do not fit the launch parameters (500 events): the
    kernels read them from the plan's page-locked image instead; results are the same,
    also after more steps than the library cycles images through."""
    rng = np.random.default_rng(11)
    lens = [int(x) for x in rng.integers(0, 40, size=500)]
    w = _w([96, 40, 0, 130, 64], [100] * 5, lens, seed=11, h_q=h_q, h_kv=2, D=D)
    db, plan = run_full(w)
    assert plan.info()["param_descriptor_bytes"] == 0
    o1 = db.out.clone()
    for _ in range(12):  # more than the images kept in flight per device
        db.release_new_pages()
        db.run_step()
    torch.cuda.synchronize()
    B.pad_device_status(db.plan)
    assert torch.equal(o1, db.out)


def test_small_batch_carries_descriptors_in_parameters():
    w = synth.tiny()
    db = DeviceBatch(w)
    plan = db.plan_step()
    n = plan.info()["param_descriptor_bytes"]
    assert 0 < n <= 8192
    db.release_new_pages(plan)


def test_status_word_reports_only_its_own_plan():
    """The status word is not reset between steps: each plan's errors are tagged with its
    generation, so a clean step on the same workspace after a failing one reports OK."""
    w = _w([200], [2], [5, 3])
    db = DeviceBatch(w)
    good = int(db.page_table[1, 0])
    db.page_table[1, 0] = w.n_pages + 5
    bad = db.run_step()
    with pytest.raises(B.PadError) as ei:
        B.pad_device_status(bad)
    assert ei.value.status == 7
    db.release_new_pages(bad)
    db.page_table[1, 0] = good
    p2 = db.run_step()
    B.pad_device_status(p2)
    torch.cuda.synchronize()
    ref_o, ref_lse = oracle.decode_step(w)
    check_outputs(db.out.cpu().numpy(), db.lse.cpu().numpy(), ref_o, ref_lse, "after a failed step")


def test_device_bounds_check_reports_bad_page():
    """A page id outside the pool in the page table is caught by the kernels' own bounds
    checks (the access is skipped) and reported through the status word."""
    w = _w([200], [2], [5, 3])
    db = DeviceBatch(w)
    db.page_table[1, 0] = w.n_pages + 5
    plan = db.run_step()
    with pytest.raises(B.PadError) as ei:
        B.pad_device_status(plan)
    assert ei.value.status == 7
    # the context stays usable
    db2 = DeviceBatch(_w([64], [1], [2]))
    p2 = db2.run_step()
    B.pad_device_status(p2)


# ---------------------------------------------------------------------------
# a4 + a5 inside the tensor-core prefix kernel
# ---------------------------------------------------------------------------

# (prefix lengths, events per video, branch lengths): 80 query rows; 140 rows with
# G = 7, so that event 18's rows 126..132 straddle two 128-row groups; a single event
_FUSED_CASES = {
    "few_events": ([4000], [3], [5, 0, 17]),
    "straddling_rows": ([3000], [20], [(7 * i) % 41 for i in range(20)]),
    "one_event_long_branch": ([6000], [1], [300]),
}


@pytest.mark.parametrize("case", sorted(_FUSED_CASES))
def test_fused_tail_and_separate_merge_both_match_oracle(case):
    prefix, epv, lens = _FUSED_CASES[case]
    w = _w(prefix, epv, lens, seed=21)
    db_f, plan_f = run_full(w, flags=B.FLAG_PREFIX_TC | B.FLAG_FUSED_MERGE, what=f"{case} fused")
    assert plan_f.info()["fused_tail"] == 1
    db_s, plan_s = run_full(w, flags=B.FLAG_PREFIX_TC, what=f"{case} separate")
    assert plan_s.info()["fused_tail"] == 0
    d = (db_f.out - db_s.out).abs().max().item()
    assert d <= 2e-3, f"fused and separate paths differ by {d:.3e}"


def test_fused_tail_same_plan_relaunched():
    """The split counters are zeroed again by the last task that reads them, so launching
    one plan again without an append (as a timing loop or a graph replay of the attention
    alone does) gives the same result; a second plan on the same workspace does too."""
    w = _w([5000], [6], [3, 9, 0, 33, 12, 4], seed=5)
    db, plan = run_full(w, flags=B.FLAG_PREFIX_TC | B.FLAG_FUSED_MERGE)
    assert plan.info()["fused_tail"] == 1
    o1 = db.out.clone()
    for _ in range(3):
        db.out.fill_(float("nan"))
        B.pad_event_decode_attn(plan, db.q, db.k_prefix, db.v_prefix, db.k_pool, db.v_pool, db.out, db.lse)
        torch.cuda.synchronize()
        B.pad_device_status(plan)
        assert torch.equal(o1, db.out)
    db.release_new_pages(plan)
    db.run_step()
    torch.cuda.synchronize()
    B.pad_device_status(db.plan)
    assert torch.equal(o1, db.out)


def test_fused_tail_wait_runs_out_and_reports_timeout():
    """A split counter that can never reach its target (set, after the append zeroed it,
    to a count no launch reaches): the tail's bounded wait gives up, the status word says
    PAD_ERR_DEVICE_TIMEOUT, and the context stays usable for the next plan."""
    w = _w([3000], [4], [5, 0, 9, 2], seed=9)
    db = DeviceBatch(w, flags=B.FLAG_PREFIX_TC | B.FLAG_FUSED_MERGE)
    plan = db.plan_step()
    info = plan.info()
    assert info["fused_tail"] == 1
    G = w.h_q // w.h_kv
    n_cnt = w.h_kv * ((4 * G + 127) // 128)
    off = info["workspace_bytes"] - (n_cnt * 4 + 255) // 256 * 256
    B.pad_kv_append(plan, db.k_new, db.v_new, db.k_pool, db.v_pool)
    db.workspace[off:off + n_cnt * 4].view(torch.int32).fill_(0x7000)
    B.pad_event_decode_attn(plan, db.q, db.k_prefix, db.v_prefix, db.k_pool, db.v_pool, db.out, db.lse)
    with pytest.raises(B.PadError) as ei:
        B.pad_device_status(plan)
    assert ei.value.status == 6
    db.release_new_pages(plan)
    p2 = db.run_step()
    B.pad_device_status(p2)
    torch.cuda.synchronize()
    ref_o, ref_lse = oracle.decode_step(w)
    check_outputs(db.out.cpu().numpy(), db.lse.cpu().numpy(), ref_o, ref_lse, "after a timed-out tail")


# ---------------------------------------------------------------------------
# pad_decode_step: a2 folded into the branch tasks
# ---------------------------------------------------------------------------

_ONE_CALL_CASES = {
    "fused_tc": (lambda: _w([4000], [3], [5, 0, 17], seed=31), B.FLAG_PREFIX_TC | B.FLAG_FUSED_MERGE),
    "separate_tc": (lambda: _w([4000], [3], [5, 0, 17], seed=31), B.FLAG_PREFIX_TC),
    "separate_tc_ragged": (lambda: _w([300, 2000, 0, 900], [5, 2, 1, 7], [16, 0, 31, 47, 2, 15, 64, 3, 9, 33,
                                                                          48, 0, 1, 16, 17], seed=32),
                           B.FLAG_PREFIX_TC),
    "mma": (lambda: synth.random_small(33, h_q=8, h_kv=2, max_events=6), B.FLAG_PREFIX_MMA),
    "simt_d64": (synth.tiny, B.FLAG_PREFIX_SIMT),
    "gqa_8k": (synth.gqa_8k, 0),
    "long_branch": (lambda: _w([700], [2], [200, 129], seed=34), B.FLAG_PREFIX_TC),
}


@pytest.mark.parametrize("case", sorted(_ONE_CALL_CASES))
def test_one_call_step_matches_two_calls(case):
    """pad_decode_step against pad_kv_append + pad_event_decode_attn on the same inputs:
    outputs, LSE, both pools and the page table bit-identical, and the oracle's
    bookkeeping and outputs met."""
    make, flags = _ONE_CALL_CASES[case]
    w = make()
    a = DeviceBatch(w, flags=flags)
    pa = a.run_step()
    b = DeviceBatch(w, flags=flags)
    pb = b.run_step(one_call=True)
    torch.cuda.synchronize()
    B.pad_device_status(pa)
    B.pad_device_status(pb)
    assert pa.info()["fused_tail"] == pb.info()["fused_tail"]
    assert torch.equal(a.out, b.out)
    assert torch.equal(a.lse, b.lse)
    assert torch.equal(a.k_pool.view(torch.int16), b.k_pool.view(torch.int16))
    assert torch.equal(a.v_pool.view(torch.int16), b.v_pool.view(torch.int16))
    assert torch.equal(a.page_table, b.page_table)
    check_bookkeeping(b, w, pb)
    ref_o, ref_lse = oracle.decode_step(w)
    check_outputs(b.out.float().cpu().numpy(), b.lse.cpu().numpy(), ref_o, ref_lse, case)


@pytest.mark.parametrize("fused", [False, True])
def test_one_call_steps_advance_like_a_generation_loop(fused):
    """Three consecutive steps through pad_decode_step, each branch one token longer than
    the last (new pages taken as lengths cross page boundaries): the pools and page table
    after the loop equal those of the same loop through the two-call path."""
    w = _w([2500], [4], [14, 15, 31, 0], seed=35)
    flags = B.FLAG_PREFIX_TC | (B.FLAG_FUSED_MERGE if fused else 0)
    a = DeviceBatch(w, flags=flags)
    b = DeviceBatch(w, flags=flags)
    lens = w.event_len.copy()
    for step in range(3):
        for db, one in ((a, False), (b, True)):
            db.plan = B.pad_plan(db.problem, db.cache, w.prefix_len, w.event_video, lens,
                                 page_table=db.page_table, max_pages=w.max_pages,
                                 workspace=db.workspace, prefix_offset=w.prefix_offset)
            if one:
                B.pad_decode_step(db.plan, db.q, db.k_new, db.v_new, db.k_prefix, db.v_prefix,
                                  db.k_pool, db.v_pool, db.out, db.lse)
            else:
                B.pad_kv_append(db.plan, db.k_new, db.v_new, db.k_pool, db.v_pool)
                B.pad_event_decode_attn(db.plan, db.q, db.k_prefix, db.v_prefix, db.k_pool,
                                        db.v_pool, db.out, db.lse)
        torch.cuda.synchronize()
        B.pad_device_status(a.plan)
        B.pad_device_status(b.plan)
        assert torch.equal(a.out, b.out) and torch.equal(a.lse, b.lse)
        lens = lens + 1
    assert torch.equal(a.page_table, b.page_table)
    assert torch.equal(a.k_pool.view(torch.int16), b.k_pool.view(torch.int16))
    assert torch.equal(a.v_pool.view(torch.int16), b.v_pool.view(torch.int16))
    assert np.array_equal(a.cache.free_pages(), b.cache.free_pages())


# ---------------------------------------------------------------------------
# Rotary embedding fused into the step (same position for a step's branches, Sec. 3.4)
# ---------------------------------------------------------------------------

_ROPE_CASES = {
    "tc_gqa_8k": (synth.gqa_8k, 0),
    "tc_ragged": (lambda: _w([300, 2000, 0, 900], [5, 2, 1, 7], [16, 0, 31, 47, 2, 15, 64, 3, 9, 33,
                                                               48, 0, 1, 16, 17], seed=42), B.FLAG_PREFIX_TC),
    "mma_small": (lambda: synth.random_small(41, h_q=8, h_kv=2, max_events=5), B.FLAG_PREFIX_MMA),
    "simt_tiny_d64": (synth.tiny, 0),
}


@pytest.mark.parametrize("one_call", [False, True])
@pytest.mark.parametrize("case", sorted(_ROPE_CASES))
def test_rope_step_matches_oracle(case, one_call):
    """q and k_new rotated at each event's step position inside the step's kernels: the
    pools hold the rotated new keys bit for bit, and the outputs match the oracle run on
    the rotated inputs."""
    make, flags = _ROPE_CASES[case]
    w = make()
    pos = synth.step_positions(w)
    table = synth.rope_table(int(pos.max()) + 8, w.head_dim)
    db = DeviceBatch(w, flags=flags)
    db.set_rope(pos, table)
    plan = db.run_step(one_call=one_call)
    torch.cuda.synchronize()
    B.pad_device_status(plan)
    wr = oracle.rotated_workload(w, pos, table)
    check_bookkeeping(db, wr, plan)
    ref_o, ref_lse = oracle.decode_step(wr)
    check_outputs(db.out.float().cpu().numpy(), db.lse.cpu().numpy(), ref_o, ref_lse, f"{case} rope")


def test_rope_at_position_zero_changes_nothing():
    """A table row of cos 1, sin 0 leaves q and k_new as they are: bit-identical to the
    step without a rotation."""
    w = _w([3000], [3], [5, 0, 17], seed=43)
    a = DeviceBatch(w)
    a.run_step(one_call=True)
    b = DeviceBatch(w)
    b.set_rope(np.zeros(w.n_events, np.int32), synth.rope_table(4, w.head_dim))
    b.run_step(one_call=True)
    torch.cuda.synchronize()
    assert torch.equal(a.out, b.out) and torch.equal(a.lse, b.lse)
    assert torch.equal(a.k_pool.view(torch.int16), b.k_pool.view(torch.int16))


# ---------------------------------------------------------------------------
# "Self G-token only" mask variant (attention ablation, Tab. 8)
# ---------------------------------------------------------------------------

def _self_g_spec(w, K=None, seed=0):
    """K per video (default: E_b + 2, at most prefix - 1) and a distinct G index per event."""
    rng = np.random.default_rng(seed)
    Ks, gi = [], np.zeros(w.n_events, np.int32)
    for b in range(w.n_videos):
        ev = w.events_of_video(b)
        k = int(K[b]) if K is not None else min(int(w.prefix_len[b]) - 1, len(ev) + 2)
        k = max(0, min(k, int(w.prefix_len[b]) - 1))
        Ks.append(k)
        if k > 0:
            pick = rng.permutation(k)
            gi[ev] = pick[np.arange(len(ev)) % k]
    return np.array(Ks, np.int32), gi


# "tc": prefix 1000 with K = 300 puts a whole 128-token split inside the planning region,
# so most rows see none of that split's keys
_SELF_G_CASES = {
    "tc_wide_planning": (lambda: _w([1000, 2600], [4, 3], [5, 0, 17, 3, 9, 1, 30], seed=51),
                         B.FLAG_PREFIX_TC, [300, 5]),
    "tc_gqa_8k": (synth.gqa_8k, 0, None),
    "mma_small": (lambda: synth.random_small(52, h_q=8, h_kv=2, max_events=5), B.FLAG_PREFIX_MMA, None),
    "mma_wide_planning": (lambda: _w([1000], [4], [5, 0, 17, 3], seed=53, h_q=8, h_kv=2),
                          B.FLAG_PREFIX_MMA, [300]),
    "simt_tiny_d64": (synth.tiny, 0, None),
    "simt_wide_planning": (lambda: _w([400], [2], [3, 9], seed=54, h_q=4, h_kv=1, D=64),
                           B.FLAG_PREFIX_SIMT, [200]),
}


@pytest.mark.parametrize("case", sorted(_SELF_G_CASES))
def test_self_g_mask_matches_oracle(case):
    make, flags, K = _SELF_G_CASES[case]
    w = make()
    Ks, gi = _self_g_spec(w, K, seed=len(case))
    db = DeviceBatch(w, flags=flags)
    db.self_g = (Ks, gi)
    plan = db.run_step(one_call=True)
    torch.cuda.synchronize()
    B.pad_device_status(plan)
    ref_o, ref_lse = oracle.decode_step(w, self_g=(Ks, gi))
    check_outputs(db.out.float().cpu().numpy(), db.lse.cpu().numpy(), ref_o, ref_lse, f"{case} self-G")
    # and it is not the default mask
    full_o, _ = oracle.decode_step(w)
    if Ks.max() > 1:
        assert np.abs(full_o - ref_o).max() > 1e-3


def test_g_all_after_self_g_is_the_default_mask():
    w = _w([3000], [3], [5, 0, 17], seed=55)
    a = DeviceBatch(w)
    a.run_step(one_call=True)
    b = DeviceBatch(w)
    plan = b.plan_step()
    Ks, gi = _self_g_spec(w)
    plan.set_g_visibility(B.G_SELF, Ks, gi)
    plan.set_g_visibility(B.G_ALL)
    B.pad_decode_step(plan, b.q, b.k_new, b.v_new, b.k_prefix, b.v_prefix, b.k_pool, b.v_pool, b.out, b.lse)
    torch.cuda.synchronize()
    assert torch.equal(a.out, b.out) and torch.equal(a.lse, b.lse)


# ---------------------------------------------------------------------------
# "Causal attention" mask variant (attention ablation, Tab. 8)
# ---------------------------------------------------------------------------

_CAUSAL_CASES = {
    "tc_ragged": (lambda: _w([300, 2000, 0, 900], [5, 2, 1, 7], [16, 0, 31, 47, 2, 15, 64, 3, 9, 33,
                                                               48, 0, 1, 16, 17], seed=61), B.FLAG_PREFIX_TC),
    "tc_many_rounds": (lambda: _w([1500], [6], [90, 70, 0, 33, 128, 1], seed=62), B.FLAG_PREFIX_TC),
    "mma_small": (lambda: synth.random_small(63, h_q=8, h_kv=2, max_events=5), B.FLAG_PREFIX_MMA),
    "simt_tiny_d64": (synth.tiny, 0),
}


@pytest.mark.parametrize("one_call", [False, True])
@pytest.mark.parametrize("case", sorted(_CAUSAL_CASES))
def test_causal_mask_matches_oracle(case, one_call):
    make, flags = _CAUSAL_CASES[case]
    w = make()
    db = DeviceBatch(w, flags=flags)
    db.causal = True
    plan = db.run_step(one_call=one_call)
    torch.cuda.synchronize()
    B.pad_device_status(plan)
    check_bookkeeping(db, w, plan)
    ref_o, ref_lse = oracle.decode_step(w, causal=True)
    check_outputs(db.out.float().cpu().numpy(), db.lse.cpu().numpy(), ref_o, ref_lse, f"{case} causal")


def test_mask_variants_and_rope_compose():
    """Causal branch visibility, the self G-token mask and the fused rotation together:
    the oracle with all three (rotated inputs, both mask changes)."""
    w = _w([1000, 2600], [4, 3], [5, 0, 17, 3, 9, 1, 30], seed=64)
    Ks, gi = _self_g_spec(w, [300, 5], seed=3)
    pos = synth.step_positions(w)
    table = synth.rope_table(int(pos.max()) + 1, w.head_dim)
    db = DeviceBatch(w, flags=B.FLAG_PREFIX_TC)
    db.causal = True
    db.self_g = (Ks, gi)
    db.set_rope(pos, table)
    plan = db.run_step(one_call=True)
    torch.cuda.synchronize()
    B.pad_device_status(plan)
    wr = oracle.rotated_workload(w, pos, table)
    check_bookkeeping(db, wr, plan)
    ref_o, ref_lse = oracle.decode_step(wr, causal=True, self_g=(Ks, gi))
    check_outputs(db.out.float().cpu().numpy(), db.lse.cpu().numpy(), ref_o, ref_lse, "all variants")
