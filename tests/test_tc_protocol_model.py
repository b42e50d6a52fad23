"""Randomised model of the tensor-core prefix kernel's mbarrier protocol.

The kernel (csrc/pad_prefix_tc.cu) runs a K producer, a V producer, an S issuer, a P.V
issuer and eight softmax warps that hand 128-token tiles to each other through
mbarriers waited on by phase parity: 3 K/V stages whose index is also the TMEM S buffer,
per-stage barriers for "K tile loaded", "V tile loaded", "S done", "P written" and "P.V
done".  A tcgen05.commit arrives when every MMA issued *by the committing thread* so far
has completed, so each issuer has its own completion barriers.  In decode, each softmax
warp owns 16 rows of the tile outright (all 128 columns), so it writes P over S columns
that no other warp reads: the warps never meet inside the loop.  In whole-sequence
prefill the two warps of a lane quarter split the columns and meet on a barrier of their
own between the row maximum and the P store; that meeting is a step inside the softmax
here (it involves no other role, and its parity alternates with the tile, like the S
buffers').

This model mirrors that schedule with asynchronous loads and MMAs that complete after
random delays and in any order, and checks under many random interleavings that no stage
or buffer is reused while something still reads it, that O is rescaled only when no P.V
is in flight, and that nothing deadlocks.  A schedule that shares one P-ready barrier and
one P.V barrier across tiles (so that a waiter can miss a phase) fails it.  TMEM is
freed only after all eight softmax warps have arrived on their own completion barrier.
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


ST = 3  # K/V stages = S buffers


MISTAKES = ("s_skips_pvfree", "k_refill_early", "v_refill_early", "rescale_without_wait",
            "dealloc_without_tdone", "one_xchg_slot")


def run(n, seed, lazy_prob=0.3, single_barriers=False, n_softmax=8, prefetch=False, meet=False,
        mistake=None):
    """prefetch: the softmax warps load tile j + 1's S during tile j (after the row maximum,
    before P(j) is released), as a softmax that hides the load behind the exponentials would.
    meet: the prefill softmax, where warps w and w + 4 (the two column halves of a lane
    quarter) exchange their partial row maxima through two shared-memory slots (tile parity)
    and a per-quarter barrier on every tile, and their row sums once more after the loop.
    mistake: one of MISTAKES, a plausible slip planted in the schedule (a wait left out, or
    one exchange slot instead of two)."""
    assert mistake is None or mistake in MISTAKES
    rnd = random.Random(seed)
    kfull = [Bar(1) for _ in range(ST)]
    vfull = [Bar(1) for _ in range(ST)]
    sfull = [Bar(1) for _ in range(ST)]
    pfull = [Bar(n_softmax) for _ in range(ST)]
    pvfree = [Bar(1) for _ in range(ST)]
    drain_s, drain_pv = Bar(1), Bar(1)
    tdone = Bar(n_softmax)
    xbar = [Bar(2) for _ in range(n_softmax // 2)]
    xslot = {}  # (slot, half, quarter) -> what the warp last wrote there
    tmem_users = [True] * n_softmax
    if single_barriers:
        pfull = [pfull[0]] * ST
        pvfree = [pvfree[0]] * ST

    def wpar(tile, per_stage=True):
        # phase parity of the completion belonging to `tile` on its barrier
        return ((tile // ST) & 1) if per_stage else (tile & 1)

    kst = [None] * ST
    vst = [None] * ST
    S_done, PV_done, P_written, PV_issued = set(), set(), set(), set()
    holding = [set() for _ in range(n_softmax)]  # tiles whose S a softmax warp has loaded, unconsumed
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

    def issue_S(t):
        def chk():
            assert kst[t % ST] == t, f"S({t}) reads a K stage not holding tile {t}"
            for j in PV_issued:
                if j % ST == t % ST and j not in PV_done:
                    raise AssertionError(f"S({t}) overwrites P({j}) still read by its P.V")
            if t >= ST:
                assert (t - ST) in PV_done, f"S({t}) before P.V({t - ST}) done"
            for h in holding:
                assert (t - ST) not in h, f"S({t}) overwrites S({t - ST}) that a softmax warp still holds"
        mma("S", chk, lambda: S_done.add(t))

    def issue_PV(j):
        def chk():
            assert j in P_written, f"P.V({j}) before P({j})"
            assert vst[j % ST] == j, f"P.V({j}) reads a V stage not holding tile {j}"
            PV_issued.add(j)
        mma("PV", chk, lambda: PV_done.add(j))

    def kprod():
        for t in range(n):
            s = t % ST
            if t >= ST and mistake != "k_refill_early":
                yield (sfull[s], ((t // ST) - 1) & 1)
            if t >= ST:
                assert (t - ST) in S_done, f"K stage reused before S({t - ST}) done"
            kst[s] = None

            def ld(t=t, s=s):
                kst[s] = t
                kfull[s].arrive()
            async_op(ld)

    def vprod():
        for t in range(n):
            s = t % ST
            if t >= ST and mistake != "v_refill_early":
                yield (pvfree[s], ((t // ST) - 1) & 1) if not single_barriers else (pvfree[s], (t - ST) & 1)
            if t >= ST:
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
            if t >= ST and mistake != "s_skips_pvfree":
                yield (pvfree[s], ((t // ST) - 1) & 1) if not single_barriers else (pvfree[s], (t - ST) & 1)
            issue_S(t)
            commit("S", sfull[s])
        commit("S", drain_s)
        yield (drain_s, 0)

    def pv_issuer():
        for j in range(n):
            s = j % ST
            yield (vfull[s], (j // ST) & 1)
            yield (pfull[s], wpar(j, not single_barriers))
            issue_PV(j)
            commit("PV", pvfree[s])
        commit("PV", drain_pv)
        yield (drain_pv, 0)

    def softmax(w):
        if prefetch and n > 0:
            yield (sfull[0], 0)
            assert 0 in S_done, "softmax loads S(0) before it is done"
            holding[w].add(0)
        for j in range(n):
            if prefetch:
                assert j in holding[w], f"softmax uses S({j}) it has not loaded"
            else:
                yield (sfull[j % ST], (j // ST) & 1)
                assert j in S_done, f"softmax reads S({j}) before it is done"
                holding[w].add(j)
            for _ in range(rnd.randint(0, 2)):  # the row maximum
                yield None
            if meet:
                yield from exchange(w, j, ("m", j))
            if prefetch and j + 1 < n:
                yield (sfull[(j + 1) % ST], ((j + 1) // ST) & 1)
                assert (j + 1) in S_done, f"softmax loads S({j + 1}) before it is done"
                holding[w].add(j + 1)
            if j > 0 and rnd.random() < lazy_prob:
                if mistake != "rescale_without_wait":
                    yield ((pvfree[(j - 1) % ST], ((j - 1) // ST) & 1) if not single_barriers
                           else (pvfree[0], (j - 1) & 1))
                assert (j - 1) in PV_done, f"O rescaled before P.V({j - 1}) done"
                for jj in PV_issued:
                    assert jj in PV_done or jj >= j, "O rescaled while a P.V is in flight"
            for _ in range(rnd.randint(0, 3)):
                yield None
            if w == 0:
                P_written.add(j)
            holding[w].discard(j)
            pfull[j % ST].arrive()
        yield (drain_pv, 0)
        assert len(PV_done) == n, "epilogue before every P.V completed"
        for _ in range(rnd.randint(0, 3)):  # reads O out of TMEM
            yield None
        if meet:
            yield from exchange(w, n, ("l", n))
        tmem_users[w] = False
        tdone.arrive()

    def exchange(w, k, tag):
        # write this half's value into slot k & 1, meet the other half (completion k of the
        # quarter's barrier), read the other half's value of the same round
        quarter, half = w % (n_softmax // 2), w // (n_softmax // 2)
        slot = 0 if mistake == "one_xchg_slot" else k & 1
        xslot[(slot, half, quarter)] = tag
        xbar[quarter].arrive()
        yield (xbar[quarter], k & 1)
        for _ in range(rnd.randint(0, 2)):
            yield None
        assert xslot.get((slot, 1 - half, quarter)) == tag, \
            f"warp {w} reads the other half's {xslot.get((slot, 1 - half, quarter))} for {tag}"

    def dealloc():
        # warp 2 frees TMEM once every softmax warp has arrived on tdone
        if mistake != "dealloc_without_tdone":
            yield (tdone, 0)
        else:
            yield (drain_pv, 0)
        assert not any(tmem_users), "TMEM freed while a softmax warp still reads it"

    actors = [kprod(), vprod(), s_issuer(), pv_issuer(), dealloc()] + [softmax(w) for w in range(n_softmax)]
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


@pytest.mark.parametrize("n", range(1, 13))
def test_prefetching_softmax_keeps_the_protocol(n):
    """Loading tile j + 1's S during tile j (waiting for its S-done barrier before releasing
    P(j)) neither deadlocks nor lets an S MMA overwrite a buffer a softmax warp still holds."""
    for seed in range(120):
        assert run(n, seed * 173 + n, prefetch=True)


@pytest.mark.parametrize("n", range(1, 13))
def test_prefill_softmax_exchange_keeps_the_protocol(n):
    """The prefill softmax's per-tile meeting of the two column halves (two slots by tile
    parity, one barrier per lane quarter) reads the other half's value of the same tile,
    and neither deadlocks nor disturbs the MMA schedule."""
    for seed in range(120):
        assert run(n, seed * 191 + n, meet=True)


@pytest.mark.parametrize("mistake", MISTAKES)
def test_model_detects_planted_mistakes(mistake):
    """Each plausible slip in the schedule (a wait dropped, or one exchange slot for both
    tile parities) fails the model under some interleaving."""
    fails = 0
    for n in range(2, 10):
        for seed in range(40):
            try:
                run(n, seed * 11 + n, lazy_prob=0.6, meet=True, mistake=mistake)
            except AssertionError:
                fails += 1
    assert fails > 0, mistake


def test_model_detects_phase_aliasing():
    fails = 0
    for n in range(4, 13):
        for seed in range(40):
            try:
                run(n, seed * 7 + n, single_barriers=True)
            except AssertionError:
                fails += 1
    assert fails > 0
