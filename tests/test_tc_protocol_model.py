import pytest
"""Randomised model of the tensor-core prefix kernel's mbarrier protocol.

The kernel (csrc/pad_prefix_tc.cu) runs a K producer, a V producer, one MMA issuer
and eight softmax warps that hand 128-token tiles to each other through mbarriers
waited on by phase parity: 3 K/V stages, 3 S buffers in TMEM (P written over S),
per-buffer P-ready barriers and P.V completions alternating over two barriers.
This model mirrors that schedule with asynchronous loads and MMAs that complete
after random delays and in any order, and checks under many random interleavings
that no stage or buffer is reused while something still reads it, that O is
rescaled only when no P.V is in flight, and that nothing deadlocks.  A schedule
with one P-ready and one P.V barrier (which lets a waiter miss a phase) fails it.
"""
import random

class Bar:
    def __init__(s, count): s.count = count; s.pending = 0; s.done = 0
    def arrive(s):
        s.pending += 1
        if s.pending == s.count: s.pending = 0; s.done += 1
    def ready(s, parity): return (s.done % 2) != parity

ST, SB = 3, 3


def run(n, seed, lazy_prob=0.3, single_barriers=False):
    rnd = random.Random(seed)
    kfull = [Bar(1) for _ in range(ST)]; vfull = [Bar(1) for _ in range(ST)]
    vempty = [Bar(1) for _ in range(ST)]; sfull = [Bar(1) for _ in range(SB)]
    pfull = [Bar(8) for _ in range(SB)]; pvdone = [Bar(1), Bar(1)]; drain = Bar(1)
    if single_barriers:
        pfull = [pfull[0]] * SB
        pvdone = [pvdone[0]] * 2
    kst = [None] * ST; vst = [None] * ST   # tile held (loaded) per stage
    S_done = set(); PV_done = set(); P_written = set(); S_issued = set(); PV_issued = set()
    inflight = []  # async ops: dict(kind, done_fn, time)
    mma_seq = []   # issued MMA op ids, to resolve commits
    now = [0]
    def async_op(fn):
        inflight.append([now[0] + rnd.randint(1, 30), fn])
    def commit(bar):
        pending = [op for op in mma_seq if not op['done']]
        if not pending: bar.arrive(); return
        ids = set(id(op) for op in pending)
        op = {'done': False, 'commit': True, 'wait': ids, 'bar': bar}
        commits.append(op)
    commits = []
    def mma(kind, t, fn_check, fn_done):
        fn_check()
        op = {'done': False}
        mma_seq.append(op)
        def fin():
            op['done'] = True; fn_done()
        async_op(fin)
    # actors as generators
    def kprod():
        for t in range(n):
            s = t % ST
            if t >= ST:
                yield (sfull[s], ((t // ST) - 1) & 1)
                assert (t - ST) in S_done, f"K stage reuse before S({t-ST}) done"
            def ld(t=t, s=s):
                kst[s] = t; kfull[s].arrive()
            kst[s] = None
            async_op(ld)
    def vprod():
        for t in range(n):
            s = t % ST
            if t >= ST:
                yield (vempty[s], ((t // ST) - 1) & 1)
                assert (t - ST) in PV_done, f"V stage reuse before PV({t-ST}) done"
            def ld(t=t, s=s):
                vst[s] = t; vfull[s].arrive()
            vst[s] = None
            async_op(ld)
    def issue_S(t):
        def chk():
            assert kst[t % ST] == t, f"S({t}) reads K stage not holding tile {t}"
            for j in PV_issued:
                if j % SB == t % SB and j not in PV_done: raise AssertionError(f"S({t}) overwrites P({j}) in flight")
            if t - SB >= 0: assert (t - SB) in PV_done, f"S({t}) before PV({t-SB}) done"
            S_issued.add(t)
        def done(): S_done.add(t)
        mma('S', t, chk, done)
    def issue_PV(j):
        def chk():
            assert j in P_written, f"PV({j}) before P({j})"
            assert vst[j % ST] == j, f"PV({j}) reads V stage not holding tile {j}"
            PV_issued.add(j)
        def done(): PV_done.add(j)
        mma('PV', j, chk, done)
    def mma_thread():
        for t in range(min(2, n)):
            yield (kfull[t % ST], (t // ST) & 1)
            issue_S(t); commit(sfull[t % SB])
        for j in range(n):
            t = j + 2
            if t < n:
                yield (kfull[t % ST], (t // ST) & 1)
                if j >= 1:
                    yield ((pvdone[(j - 1) & 1], ((j - 1) >> 1) & 1) if not single_barriers
                           else (pvdone[0], (j - 1) & 1))
                issue_S(t); commit(sfull[t % SB])
            s = j % ST
            yield (vfull[s], (j // ST) & 1)
            yield (pfull[j % SB], (j // SB) & 1) if not single_barriers else (pfull[0], j & 1)
            issue_PV(j); commit(pvdone[j & 1]); commit(vempty[s])
        commit(drain)
        yield (drain, 0)
    def softmax(w):
        for j in range(n):
            yield (sfull[j % SB], (j // SB) & 1)
            assert j in S_done, f"softmax reads S({j}) before done"
            if j > 0 and rnd.random() < lazy_prob:
                yield ((pvdone[(j - 1) & 1], ((j - 1) >> 1) & 1) if not single_barriers
                       else (pvdone[0], (j - 1) & 1))
                assert (j - 1) in PV_done, f"rescale before PV({j-1}) done"
                for jj in PV_issued:
                    assert jj in PV_done or jj >= j, "O written while rescaling"
            for _ in range(rnd.randint(0, 3)): yield None
            P_written.add(j) if w == 0 else None
            pfull[j % SB].arrive()
        yield (drain, 0)
        assert len(PV_done) == n, "epilogue before all P.V done"
    actors = [kprod(), vprod(), mma_thread()] + [softmax(w) for w in range(8)]
    waiting = [None] * len(actors); alive = [True] * len(actors)
    # P_written must be set before any of the 4 arrivals completes the barrier: mark at first
    steps = 0
    while any(alive):
        steps += 1
        if steps > 200000: raise AssertionError("no progress (deadlock)")
        now[0] += 1
        # complete async ops
        rnd.shuffle(inflight)
        for op in list(inflight):
            if op[0] <= now[0] and rnd.random() < 0.7:
                inflight.remove(op); op[1]()
        for c in list(commits):
            if all(o['done'] for o in mma_seq if id(o) in c['wait']):
                commits.remove(c); c['bar'].arrive()
        order = list(range(len(actors))); rnd.shuffle(order)
        progressed = False
        for i in order:
            if not alive[i]: continue
            if waiting[i] is not None:
                bar, par = waiting[i]
                if not bar.ready(par): continue
                waiting[i] = None
            if rnd.random() < 0.5: continue
            try:
                w = next(actors[i])
                if w is not None: waiting[i] = w
                progressed = True
            except StopIteration:
                alive[i] = False
        if any(alive) and not progressed and not inflight and not commits and all(
                (not alive[i]) or (waiting[i] is not None and not waiting[i][0].ready(waiting[i][1]))
                for i in range(len(actors))):
            raise AssertionError(f"deadlock at n={n}")
    return True



@pytest.mark.parametrize("n", range(1, 13))
def test_tc_kernel_barrier_protocol(n):
    for seed in range(150):
        assert run(n, seed * 131 + n)


def test_model_detects_phase_aliasing():
    fails = 0
    for n in range(4, 13):
        for seed in range(40):
            try:
                run(n, seed * 7 + n, single_barriers=True)
            except AssertionError:
                fails += 1
    assert fails > 0
