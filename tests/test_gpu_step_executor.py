"""The step executor (pad_step_*), the host runtime of a serving loop: one call per step.

Its runs must be the library's own step calls, bit for bit: outputs, LSE, both pools and the
page table against pad_plan + pad_decode_step (and + pad_kv_append + pad_event_decode_attn
for the two-call option), the host-buffer run against the device-buffer run, and a
generation loop that advances event_len in place against the same loop through pad_plan.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_02963_gb300 import binding as B
from paper_2607_02963_gb300 import synth
from paper_2607_02963_gb300.device import DeviceBatch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda(padlib):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.init()


def _native(db, w, stream=None, **kw):
    return B.NativeStep(db.problem, db.cache, w.prefix_len, w.event_video, w.event_len, db.page_table,
                        w.max_pages, db.workspace, w.prefix_offset, db.q, db.k_new, db.v_new, db.k_prefix,
                        db.v_prefix, db.k_pool, db.v_pool, db.out, db.lse,
                        stream if stream is not None else torch.cuda.current_stream(), **kw)


def _same_state(a, b):
    assert torch.equal(a.out, b.out) and torch.equal(a.lse, b.lse)
    assert torch.equal(a.k_pool.view(torch.int16), b.k_pool.view(torch.int16))
    assert torch.equal(a.v_pool.view(torch.int16), b.v_pool.view(torch.int16))
    assert torch.equal(a.page_table, b.page_table)


@pytest.mark.parametrize("one_call", [True, False])
@pytest.mark.parametrize("make", [synth.gqa_8k, lambda: synth.random_small(5), synth.tiny, synth.long_32k])
def test_run_matches_the_step_calls(make, one_call):
    """The executor (pad_step_run, the call the bench times) against pad_plan plus the step
    calls: the same outputs, pools and page table, and the oracle's outputs (long_32k: the
    plan whose branch tasks wait for the prefix grid first)."""
    w = make()
    a = DeviceBatch(w)
    pa = a.run_step(one_call=one_call)
    b = DeviceBatch(w)
    st = _native(b, w, release_pages=False, one_call=one_call)
    st()
    torch.cuda.synchronize()
    B.pad_device_status(pa)
    _same_state(a, b)
    assert np.array_equal(st.new_page, pa.new_pages())
    ref_o, ref_lse = oracle.decode_step(w)
    got = b.out.float().cpu().numpy()
    assert np.abs(got - ref_o).max() <= 1e-2


@pytest.mark.parametrize("adjacent", [True, False])
def test_run_host_copies_in_and_out(adjacent):
    """Host buffers laid out like the device ones (one copy each way) or apart (five)."""
    w = synth.gqa_8k()
    a = DeviceBatch(w)
    a.run_step(one_call=True)
    torch.cuda.synchronize()
    b = DeviceBatch(w)
    if adjacent:
        h_in = b.io_in.cpu().pin_memory()
        h_out = torch.empty(b.io_out.shape, dtype=torch.uint8).pin_memory()
        qn, kn = b.q.numel(), b.k_new.numel()
        hq, hk, hv = h_in[:qn].view(b.q.shape), h_in[qn:qn + kn].view(b.k_new.shape), h_in[qn + kn:].view(b.v_new.shape)
        ob = b.out.numel() * b.out.element_size()
        ho = h_out[:ob].view(b.out.dtype).view(b.out.shape)
        hl = h_out[ob:].view(torch.float32).view(b.lse.shape)
    else:
        hq = b.q.cpu().pin_memory()
        hk = b.k_new.cpu().pin_memory()
        hv = b.v_new.cpu().pin_memory()
        ho = torch.empty(b.out.shape, dtype=b.out.dtype).pin_memory()
        hl = torch.empty(b.lse.shape, dtype=torch.float32).pin_memory()
    b.q.zero_()
    b.k_new.zero_()
    b.v_new.zero_()
    st = _native(b, w, release_pages=False)
    st.run_host(hq, hk, hv, ho, hl)
    assert torch.equal(ho, a.out.cpu()) and torch.equal(hl, a.lse.cpu())
    _same_state(a, b)


@pytest.mark.parametrize("one_call", [True, False])
@pytest.mark.parametrize("adjacent", [True, False])
@pytest.mark.parametrize("make", [synth.gqa_8k, synth.tiny])
def test_run_host_mapped_io(make, adjacent, one_call):
    """Mapped host I/O: a kernel reads q / k_new / v_new from the page-locked buffers and the
    step writes O and LSE straight into them; the results, pools and page table equal the
    device-buffer run bit for bit, and the step's own device out / lse stay untouched."""
    w = make()
    a = DeviceBatch(w)
    a.run_step(one_call=one_call)
    torch.cuda.synchronize()
    b = DeviceBatch(w)
    if adjacent:
        h_in = b.io_in.cpu().pin_memory()
        h_out = torch.full(b.io_out.shape, 0x7f, dtype=torch.uint8).pin_memory()
        qn, kn = b.q.numel(), b.k_new.numel()
        hq, hk, hv = h_in[:qn].view(b.q.shape), h_in[qn:qn + kn].view(b.k_new.shape), h_in[qn + kn:].view(b.v_new.shape)
        ob = b.out.numel() * b.out.element_size()
        ho = h_out[:ob].view(b.out.dtype).view(b.out.shape)
        hl = h_out[ob:].view(torch.float32).view(b.lse.shape)
    else:
        hq = b.q.cpu().pin_memory()
        hk = b.k_new.cpu().pin_memory()
        hv = b.v_new.cpu().pin_memory()
        ho = torch.full(b.out.shape, float("nan"), dtype=b.out.dtype).pin_memory()
        hl = torch.full(b.lse.shape, float("nan"), dtype=torch.float32).pin_memory()
    b.q.zero_()
    b.k_new.zero_()
    b.v_new.zero_()
    b.out.fill_(7.0)
    b.lse.fill_(7.0)
    st = _native(b, w, release_pages=False, one_call=one_call, mapped_host_io=True)
    st.profile(True)
    st.run_host(hq, hk, hv, ho, hl)
    prof = st.profile_read()
    assert prof["calls"] == 1
    assert torch.equal(ho, a.out.cpu()) and torch.equal(hl, a.lse.cpu())
    # inputs landed in the device buffers; outputs went to the host only
    assert torch.equal(b.q.cpu(), a.q.cpu()) and torch.equal(b.k_new.cpu(), a.k_new.cpu())
    assert torch.equal(b.v_new.cpu(), a.v_new.cpu())
    assert bool((b.out == 7.0).all()) and bool((b.lse == 7.0).all())
    assert torch.equal(a.k_pool.view(torch.int16), b.k_pool.view(torch.int16))
    assert torch.equal(a.v_pool.view(torch.int16), b.v_pool.view(torch.int16))
    assert torch.equal(a.page_table, b.page_table)


@pytest.mark.parametrize("own_stream", [False, True])
@pytest.mark.parametrize("mapped", [True, False])
def test_two_batches_in_flight(mapped, own_stream):
    """pad_step_enqueue_host of two independent batches, then pad_step_wait of each: every
    batch's outputs and state equal its own device-buffer run.  With own_stream the second
    batch's executor runs on a stream of its own (how the bench keeps two batches in flight),
    so the two batches' kernels and host reads and writes may overlap."""
    ws = [synth.long_32k() if own_stream else synth.gqa_8k(), synth.random_small(3)]
    refs, runs, bufs = [], [], []
    for w in ws:
        a = DeviceBatch(w)
        a.run_step(one_call=True)
        refs.append(a)
    torch.cuda.synchronize()
    for w in ws:
        b = DeviceBatch(w)
        hq, hk, hv = b.q.cpu().pin_memory(), b.k_new.cpu().pin_memory(), b.v_new.cpu().pin_memory()
        ho = torch.empty(b.out.shape, dtype=b.out.dtype).pin_memory()
        hl = torch.empty(b.lse.shape, dtype=torch.float32).pin_memory()
        b.q.zero_()
        stream = torch.cuda.Stream() if own_stream and len(runs) == 1 else None
        runs.append((b, _native(b, w, stream=stream, release_pages=False, mapped_host_io=mapped)))
        bufs.append((hq, hk, hv, ho, hl))
    for (b, st), io in zip(runs, bufs):
        st.enqueue_host(*io)
    runs[1][1].wait()
    runs[0][1].wait()
    runs[0][1].wait()  # nothing pending: returns at once
    for a, (b, st), io in zip(refs, runs, bufs):
        assert torch.equal(io[3], a.out.cpu()) and torch.equal(io[4], a.lse.cpu())
        assert torch.equal(a.page_table, b.page_table)
        assert torch.equal(a.k_pool.view(torch.int16), b.k_pool.view(torch.int16))


@pytest.mark.parametrize("mapped", [True, False])
def test_two_steps_of_one_executor_in_flight(mapped):
    """Two consecutive steps of one generation loop enqueued back to back on one executor
    (their own host buffers, no wait in between): the second step's inputs reach the device
    only after the first step's kernels have read theirs, so both steps' outputs, the pools
    and the page table equal the same two steps run one after the other."""
    w = synth.make_workload("two", 21, 28, 4, 128, [3000], [6], [15, 16, 31, 0, 47, 8],
                            rng=np.random.default_rng(21))
    rng = np.random.default_rng(5)
    ins = [[torch.from_numpy(rng.standard_normal(t.shape).astype(np.float32)).to(torch.bfloat16)
            for t in (w.q, w.k_new, w.v_new)] for _ in range(2)]
    # reference: two serial steps
    a = DeviceBatch(w)
    sa = _native(a, w, release_pages=False, mapped_host_io=mapped)
    ref = []
    for k in range(2):
        hq, hk, hv = (x.pin_memory() for x in ins[k])
        ho = torch.empty(a.out.shape, dtype=a.out.dtype).pin_memory()
        hl = torch.empty(a.lse.shape, dtype=torch.float32).pin_memory()
        sa.run_host(hq, hk, hv, ho, hl)
        ref.append((ho.clone(), hl.clone()))
        sa.event_len += 1
    # the same two steps in flight
    b = DeviceBatch(w)
    sb = _native(b, w, release_pages=False, mapped_host_io=mapped)
    outs = []
    for k in range(2):
        hq, hk, hv = (x.pin_memory() for x in ins[k])
        ho = torch.full(b.out.shape, float("nan"), dtype=b.out.dtype).pin_memory()
        hl = torch.full(b.lse.shape, float("nan"), dtype=torch.float32).pin_memory()
        sb.enqueue_host(hq, hk, hv, ho, hl)
        outs.append((hq, hk, hv, ho, hl))
        sb.event_len += 1
    sb.wait()
    torch.cuda.synchronize()
    for k in range(2):
        assert torch.equal(outs[k][3], ref[k][0]) and torch.equal(outs[k][4], ref[k][1])
    assert torch.equal(a.k_pool.view(torch.int16), b.k_pool.view(torch.int16))
    assert torch.equal(a.v_pool.view(torch.int16), b.v_pool.view(torch.int16))
    assert torch.equal(a.page_table, b.page_table)


def test_run_host_mapped_io_falls_back_on_pageable_buffers():
    """A pageable host buffer fails the mapped check: that call takes the copy path."""
    w = synth.tiny()
    a = DeviceBatch(w)
    a.run_step(one_call=True)
    torch.cuda.synchronize()
    b = DeviceBatch(w)
    hq = b.q.cpu()  # pageable
    hk = b.k_new.cpu().pin_memory()
    hv = b.v_new.cpu().pin_memory()
    ho = torch.empty(b.out.shape, dtype=b.out.dtype).pin_memory()
    hl = torch.empty(b.lse.shape, dtype=torch.float32).pin_memory()
    b.q.zero_()
    st = _native(b, w, release_pages=False, mapped_host_io=True)
    st.run_host(hq, hk, hv, ho, hl)
    assert torch.equal(ho, a.out.cpu()) and torch.equal(hl, a.lse.cpu())
    _same_state(a, b)  # the copy path also writes the step's device out / lse


@pytest.mark.parametrize("one_call", [True, False])
def test_generation_loop_advances_event_len_in_place(one_call):
    """Three steps; each run plans from the executor's event_len as the loop left it."""
    w = synth.make_workload("loop", 61, 28, 4, 128, [2500], [4], [14, 15, 31, 0],
                            rng=np.random.default_rng(61))
    a = DeviceBatch(w)
    b = DeviceBatch(w)
    st = _native(b, w, release_pages=False, one_call=one_call)
    lens = w.event_len.copy()
    for step in range(3):
        a.plan = B.pad_plan(a.problem, a.cache, w.prefix_len, w.event_video, lens, page_table=a.page_table,
                            max_pages=w.max_pages, workspace=a.workspace, prefix_offset=w.prefix_offset)
        B.pad_decode_step(a.plan, a.q, a.k_new, a.v_new, a.k_prefix, a.v_prefix, a.k_pool, a.v_pool, a.out, a.lse)
        st.event_len[:] = lens
        st()
        torch.cuda.synchronize()
        B.pad_device_status(a.plan)
        assert np.array_equal(st.new_page, a.plan.new_pages())
        _same_state(a, b)
        lens = lens + 1
    assert np.array_equal(a.cache.free_pages(), b.cache.free_pages())
