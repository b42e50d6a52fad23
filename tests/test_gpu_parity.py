"""Parity of the CUDA path (through the C ABI) against the fp64 oracle.

Bar (from the problem statement): page-table and pool bookkeeping bit-exact;
outputs within max-abs <= 1e-2 and relative-L2 <= 2e-3 (bf16 in, fp32
accumulate); the natural-log LSE within 1e-3 absolute (a log of an fp32 sum of
positive terms: its error is the relative error of that sum, ~1e-6 here).
"""
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


def run_full(w, flags=0, out_dtype=0, what=""):
    db = DeviceBatch(w, flags=flags, out_dtype=out_dtype)
    plan = db.run_step()
    torch.cuda.synchronize()
    B.pad_device_status(plan)
    check_bookkeeping(db, w, plan)
    ref_o, ref_lse = oracle.decode_step(w)
    got = db.out.float().cpu().numpy()
    check_outputs(got, db.lse.cpu().numpy(), ref_o, ref_lse, what or w.name)
    return db, plan


def run_sampled(w, events, heads=None, flags=0, what=""):
    """Full-size step; the oracle computes the sampled events one by one."""
    db = DeviceBatch(w, flags=flags)
    plan = db.run_step()
    torch.cuda.synchronize()
    B.pad_device_status(plan)
    check_bookkeeping(db, w, plan)
    got_o = db.out.cpu().numpy()
    got_l = db.lse.cpu().numpy()
    for e in events:
        ro, rl = oracle.event_rows(w, int(e), heads)
        go = got_o[e] if heads is None else got_o[e, heads]
        gl = got_l[e] if heads is None else got_l[e, heads]
        check_outputs(go, gl, ro, rl, f"{what or w.name} event {e}")
    return db, plan


# ---------------------------------------------------------------------------
# The five workloads
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("flags", [0, B.FLAG_PREFIX_SIMT, B.FLAG_PREFIX_MMA])
def test_tiny_full(flags):
    run_full(synth.tiny(), flags=flags)


@pytest.mark.parametrize("flags", [0, B.FLAG_PREFIX_MMA, B.FLAG_PREFIX_TC])
def test_gqa_8k_full(flags):
    run_full(synth.gqa_8k(), flags=flags)


@pytest.mark.parametrize("flags", [0, B.FLAG_PREFIX_TC])
def test_long_32k_sampled(flags):
    w = synth.long_32k()
    rng = np.random.default_rng(0)
    ev = sorted(set([0, w.n_events - 1] + list(rng.choice(w.n_events, 4, replace=False))))
    run_sampled(w, ev, flags=flags)


@pytest.mark.parametrize("flags", [0, B.FLAG_PREFIX_TC])
def test_ragged_serving_sampled(flags):
    w = synth.ragged_serving()
    ev = []
    for b in range(w.n_videos):
        idx = w.events_of_video(b)
        ev += [int(idx[0]), int(idx[-1])] if b % 3 == 0 else [int(idx[len(idx) // 2])]
    run_sampled(w, sorted(set(ev)), flags=flags)


@pytest.mark.parametrize("E", synth.SWEEP_E)
@pytest.mark.parametrize("flags", [0, B.FLAG_PREFIX_TC])
def test_event_sweep_sampled(E, flags):
    w = synth.event_sweep(E)
    ev = sorted(set([0, E - 1, E // 2]))
    run_sampled(w, ev, flags=flags)


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
def test_random_small_simt(seed):
    run_full(synth.random_small(seed, h_q=8, h_kv=2, max_prefix=900, max_events=4),
             flags=B.FLAG_PREFIX_SIMT)


@pytest.mark.parametrize("seed", range(3))
def test_random_small_head_dim_64(seed):
    w = synth.random_small(50 + seed, h_q=16, h_kv=4, head_dim=64, max_prefix=600, max_events=4)
    run_full(w, flags=B.FLAG_PREFIX_MMA)
    run_full(w, flags=B.FLAG_PREFIX_SIMT)


@pytest.mark.parametrize("flags", [B.FLAG_PREFIX_MMA, B.FLAG_PREFIX_TC])
def test_large_group_and_outlier_channels(flags):
    w = synth.random_small(60, h_q=32, h_kv=2, max_prefix=700, max_events=3, k_scale_sigma=0.5)
    run_full(w, flags=flags)


# ---------------------------------------------------------------------------
# Edge cases
# ---------------------------------------------------------------------------

def _w(prefix, epv, lens, seed=7, h_q=28, h_kv=4, D=128, sigma=None):
    rng = np.random.default_rng(seed)
    return synth.make_workload("edge", seed, h_q, h_kv, D, prefix, epv, lens, rng=rng,
                               k_scale_sigma=sigma)


@pytest.mark.parametrize("flags", [B.FLAG_PREFIX_SIMT, B.FLAG_PREFIX_MMA, B.FLAG_PREFIX_TC])
def test_single_event_empty_branch(flags):
    run_full(_w([300], [1], [0]), flags=flags)          # query sees the prefix and itself


@pytest.mark.parametrize("lens", [[16, 32, 0, 15, 17], [1, 31, 48, 63, 64]])
def test_page_boundaries(lens):
    run_full(_w([257], [len(lens)], lens))


@pytest.mark.parametrize("flags", [B.FLAG_PREFIX_MMA, B.FLAG_PREFIX_TC])
def test_prefix_not_multiple_of_tile_and_tiny_prefix(flags):
    run_full(_w([1, 129, 65], [2, 3, 2], [3, 0, 9, 16, 2, 5, 7]), flags=flags)


@pytest.mark.parametrize("flags", [B.FLAG_PREFIX_MMA, B.FLAG_PREFIX_TC])
def test_video_with_empty_prefix_and_video_without_events(flags):
    run_full(_w([0, 500, 200], [2, 0, 3], [4, 1, 0, 16, 2]), flags=flags)


@pytest.mark.parametrize("flags", [B.FLAG_PREFIX_MMA, B.FLAG_PREFIX_TC])
def test_sixty_four_events(flags):
    run_full(_w([700], [64], list(np.arange(64) % 40)), flags=flags)


def test_long_split_many_tiles_tc():
    """Few SMs -> long splits: many 64-token tiles per CTA (the 4-stage ring wraps several
    times, both S buffers alternate, lazy rescaling meets growing maxima)."""
    w = _w([5000, 3001], [5, 9], list(range(0, 70, 5)), sigma=0.5)
    db = DeviceBatch(w, flags=B.FLAG_PREFIX_TC, num_sms=4)
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
    ev = [0, 99, 100, 250, 299, 300, 401, 499]
    db, plan = run_sampled(w, ev)
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
