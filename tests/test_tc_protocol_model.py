"""Randomised model of the tensor-core prefix kernel's mbarrier protocol.

The kernel (csrc/pad_prefix_tc.cu) runs a K producer, a V producer, an S issuer, a P.V
issuer and eight softmax warps that hand 128-token tiles to each other through
mbarriers waited on by phase parity: 3 K/V stages ("K tile loaded", "V tile loaded",
"S of the tile in this K stage done", "P.V of the tile in this V stage done"), one TMEM
S buffer ("S done", "S loaded by every softmax warp") and two TMEM P slots ("P written").
The two key halves of a tile (tokens 0-63: softmax warps 0-3 here, 64-127: warps 4-7)
keep their own softmax state and P.V accumulator: the first four P.V MMAs of a tile add
into O_A, the last four into O_B, and a warp rescales only its own half's O.  A
tcgen05.commit arrives when every MMA issued *by the committing thread* so far has
completed, so each issuer has its own completion barriers.

This model mirrors that schedule with asynchronous loads and MMAs that complete after
random delays and in any order, and checks under many random interleavings that no stage,
buffer or slot is reused while something still reads it, that an O accumulator is
rescaled only when no P.V into it is in flight, and that nothing deadlocks.  Schedules
with a plausible mistake fail it: one that shares one P-ready barrier and one P.V barrier
across tiles, one that issues the next S before every softmax warp has loaded the current
one, and one that writes P into a slot before the P.V of two tiles back has read it.  TMEM
is freed only after all eight softmax warps have arrived on their own completion barrier.
"""
import random

import pytest


class Bar:
    def __init__(s, count):
        s.count = count
        s.pending = 0
        s.done = 0

    def arrive(s):
        s.pending += 1
        if s.pending == s.count:
            s.pending = 0
            s.done += 1

    def ready(s, parity):
        return (s.done % 2) != parity


ST = 3  # K/V stages
PS = 2  # TMEM P slots
N_SOFTMAX = 8  # warps 0-3: key half A, 4-7: key half B


def run(n, seed, lazy_prob=0.3, single_barriers=False, s_before_loaded=False, p_slot_unchecked=False):
    rnd = random.Random(seed)
    kfull = [Bar(1) for _ in range(ST)]
    vfull = [Bar(1) for _ in range(ST)]
    kfree = [Bar(1) for _ in range(ST)]
    pvfree = [Bar(1) for _ in range(ST)]
    sfull = Bar(1)
    sfree = Bar(N_SOFTMAX)
    pfull = [Bar(N_SOFTMAX) for _ in range(PS)]
    drain_s, drain_pv = Bar(1), Bar(1)
    tdone = Bar(N_SOFTMAX)
    xchg = Bar(N_SOFTMAX)
    tmem_users = [True] * N_SOFTMAX
    if single_barriers:
        pfull = [pfull[0]] * PS
        pvfree = [pvfree[0]] * ST

    kst = [None] * ST
    vst = [None] * ST
    S_done, PV_done = set(), set()
    P_written = {}                 # tile -> halves whose P is written
    PV_issued = set()
    pv_inflight = {0: 0, 1: 0}     # P.V MMAs into O_A / O_B not yet complete
    holding = [set() for _ in range(N_SOFTMAX)]  # tiles whose S a softmax warp still reads
    inflight = []
    commits = []
    issued = {"S": [], "PV": []}  # per-issuer MMA ops (a commit tracks only its own)
    now = [0]

    def async_op(fn):
        inflight.append([now[0] + rnd.randint(1, 30), fn])

    def commit(who, bar):
        pend = [op for op in issued[who] if not op["done"]]
        if not pend:
            bar.arrive()
            return
        commits.append({"wait": pend, "bar": bar})

    def mma(who, check, done):
        check()
        op = {"done": False}
        issued[who].append(op)

        def fin():
            op["done"] = True
            done()
        async_op(fin)

    pv_half_done = {}

    def issue_S(t):
        def chk():
            assert kst[t % ST] == t, f"S({t}) reads a K stage not holding tile {t}"
            for h in holding:
                for j in h:
                    if j != t:
                        raise AssertionError(f"S({t}) overwrites S({j}) that a softmax warp still loads")
        mma("S", chk, lambda: S_done.add(t))

    def issue_PV(j, half):
        # the four MMAs of one key half, into that half's accumulator
        def chk():
            assert half in P_written.get(j, set()), f"P.V({j}) half {half} before its P"
            assert vst[j % ST] == j, f"P.V({j}) reads a V stage not holding tile {j}"
            PV_issued.add(j)
            pv_inflight[half] += 1

        def done():
            pv_inflight[half] -= 1
            pv_half_done[j] = pv_half_done.get(j, 0) + 1
            if pv_half_done[j] == 2:
                PV_done.add(j)
        mma("PV", chk, done)

    def kprod():
        for t in range(n):
            s = t % ST
            if t >= ST:
                yield (kfree[s], ((t // ST) - 1) & 1)
                assert (t - ST) in S_done, f"K stage reused before S({t - ST}) done"
            kst[s] = None

            def ld(t=t, s=s):
                kst[s] = t
                kfull[s].arrive()
            async_op(ld)

    def pv_wait(tile):
        # the completion of P.V(tile) on its V stage's barrier
        if single_barriers:
            return (pvfree[0], tile & 1)
        return (pvfree[tile % ST], (tile // ST) & 1)

    def vprod():
        for t in range(n):
            s = t % ST
            if t >= ST:
                yield pv_wait(t - ST)
                assert (t - ST) in PV_done, f"V stage reused before P.V({t - ST}) done"
            vst[s] = None

            def ld(t=t, s=s):
                vst[s] = t
                vfull[s].arrive()
            async_op(ld)

    def s_issuer():
        for t in range(n):
            s = t % ST
            yield (kfull[s], (t // ST) & 1)
            if t >= 1 and not s_before_loaded:
                yield (sfree, (t - 1) & 1)  # every softmax warp has loaded S(t - 1)
            issue_S(t)
            commit("S", sfull)
            commit("S", kfree[s])
        commit("S", drain_s)
        yield (drain_s, 0)

    def pv_issuer():
        for j in range(n):
            s = j % ST
            yield (vfull[s], (j // ST) & 1)
            yield (pfull[0], j & 1) if single_barriers else (pfull[j % PS], (j // PS) & 1)
            issue_PV(j, 0)
            issue_PV(j, 1)
            commit("PV", pvfree[s])
        commit("PV", drain_pv)
        yield (drain_pv, 0)

    p_count = {}

    def softmax(w):
        half = w // (N_SOFTMAX // 2)
        for j in range(n):
            yield (sfull, j & 1)
            assert j in S_done, f"softmax reads S({j}) before it is done"
            holding[w].add(j)
            for _ in range(rnd.randint(0, 2)):  # S load
                yield None
            holding[w].discard(j)
            sfree.arrive()
            for _ in range(rnd.randint(0, 2)):  # row maximum
                yield None
            if j > 0 and rnd.random() < lazy_prob:
                yield pv_wait(j - 1)
                assert (j - 1) in PV_done, f"O rescaled before P.V({j - 1}) done"
                assert pv_inflight[half] == 0, "O rescaled while a P.V into it is in flight"
            if j >= PS and not p_slot_unchecked:
                yield pv_wait(j - PS)  # P slot j % 2 held P(j - 2) until its P.V completed
            for jj in PV_issued:
                if jj % PS == j % PS and jj != j and jj not in PV_done:
                    raise AssertionError(f"P({j}) overwrites P({jj}) still read by its P.V")
            for _ in range(rnd.randint(0, 3)):  # exponentials
                yield None
            key = (j, half)
            p_count[key] = p_count.get(key, 0) + 1
            if p_count[key] == N_SOFTMAX // 2:
                P_written.setdefault(j, set()).add(half)
            pfull[j % PS].arrive()
        yield (drain_pv, 0)
        assert len(PV_done) == n, "epilogue before every P.V completed"
        # the two halves meet once, then each merges both accumulators
        xchg.arrive()
        yield (xchg, 0)
        for _ in range(rnd.randint(0, 3)):  # reads O_A and O_B out of TMEM
            yield None
        tmem_users[w] = False
        tdone.arrive()

    def dealloc():
        # warp 2 frees TMEM once every softmax warp has arrived on tdone
        yield (tdone, 0)
        assert not any(tmem_users), "TMEM freed while a softmax warp still reads it"

    actors = [kprod(), vprod(), s_issuer(), pv_issuer(), dealloc()] + [softmax(w) for w in range(N_SOFTMAX)]
    waiting = [None] * len(actors)
    alive = [True] * len(actors)
    steps = 0
    while any(alive):
        steps += 1
        if steps > 400000:
            raise AssertionError("no progress")
        now[0] += 1
        rnd.shuffle(inflight)
        for op in list(inflight):
            if op[0] <= now[0] and rnd.random() < 0.7:
                inflight.remove(op)
                op[1]()
        for c in list(commits):
            if all(o["done"] for o in c["wait"]):
                commits.remove(c)
                c["bar"].arrive()
        order = list(range(len(actors)))
        rnd.shuffle(order)
        progressed = False
        for i in order:
            if not alive[i]:
                continue
            if waiting[i] is not None:
                bar, par = waiting[i]
                if not bar.ready(par):
                    continue
                waiting[i] = None
            if rnd.random() < 0.5:
                continue
            try:
                w = next(actors[i])
                if w is not None:
                    waiting[i] = w
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
    for seed in range(120):
        assert run(n, seed * 131 + n)


def _fails(**kw):
    fails = 0
    for n in range(3, 13):
        for seed in range(40):
            try:
                run(n, seed * 7 + n, **kw)
            except AssertionError:
                fails += 1
    return fails


def test_model_detects_phase_aliasing():
    assert _fails(single_barriers=True) > 0


def test_model_detects_s_issued_before_every_warp_loaded_the_last():
    assert _fails(s_before_loaded=True) > 0


def test_model_detects_p_slot_reuse_before_its_pv():
    assert _fails(p_slot_unchecked=True) > 0
