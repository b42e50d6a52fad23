"""Randomised model of the dual prefix kernel's mbarrier protocol (csrc/pad_prefix_dual.cu).

The kernel runs a TMA producer, an S issuer, a P.V issuer and two softmax groups (slots)
that hand 128-token tiles to each other through mbarriers waited on by phase parity.  With
two row groups every tile is used by both slots (S_g = Q_g K^T, O_g += P_g V); with one row
group the slots take alternate tiles.  K tiles live in 3 stages, V tiles in 2 (3 with one
row group), each slot has one TMEM S buffer whose first half receives P, and the P.V of a
tile runs in two halves, each released by its own P-written barrier.  A tcgen05.commit
arrives when every MMA issued *by the committing thread* so far has completed.  At the end
each group stages its O rows in shared memory the MMAs no longer read: slot 0 of two row
groups in the K stages, slot 1 in the V stages, one row group in the K stages.

The model runs the same schedule with loads and MMAs that complete after random delays, and
checks under many random interleavings that no stage or buffer is overwritten while a load
lands in it or something still reads it, that O is rescaled only when no P.V into it is in
flight, and that nothing deadlocks.  It finds the hazard of staging slot 0's rows before the
S issuer's last MMA (slot 1's) has finished reading the K stages.
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


KS = 3


def run(n_tiles, dual, seed, lazy_prob=0.3, stage_without_drain=False, n_warps=4):
    rnd = random.Random(seed)
    VS = 2 if dual else 3
    n_slot = [n_tiles, n_tiles] if dual else [(n_tiles + 1) // 2, n_tiles // 2]
    n_seq = sum(n_slot)

    def seq(i):
        g, k = i & 1, i >> 1
        return g, k, (k if dual else i)

    kfull = [Bar(1) for _ in range(KS)]
    kfree = [Bar(1) for _ in range(KS)]
    vfull = [Bar(1) for _ in range(3)]
    vfree = [Bar(1) for _ in range(3)]
    sfull = [Bar(1) for _ in range(2)]
    plo = [Bar(n_warps) for _ in range(2)]
    phi = [Bar(n_warps) for _ in range(2)]
    pvlo = [Bar(1) for _ in range(2)]
    pvdone = [Bar(1) for _ in range(2)]
    drain_s, drain_pv = Bar(1), Bar(1)

    kst = [-1] * KS         # tile held by each K stage (-1: never loaded; None: a load is landing)
    vst = [-1] * 3
    reading = []            # in-flight MMAs: dicts with the regions they read
    s_buf = [None, None]    # tile whose S (or P) the slot's S buffer holds
    p_half = [set(), set()]  # halves of P written for the current tile of the slot
    pv_inflight = [0, 0]    # P.V MMAs into O_g not yet complete
    holding = [set(), set()]  # (slot, tile) S values a softmax warp still reads
    inflight = []
    commits = []
    issued = {"S": [], "PV": []}
    now = [0]

    def async_op(fn):
        inflight.append([now[0] + rnd.randint(1, 30), fn])

    def commit(who, bar):
        pend = [op for op in issued[who] if not op["done"]]
        if not pend:
            bar.arrive()
        else:
            commits.append({"wait": pend, "bar": bar})

    def mma(who, regions, check, done):
        check()
        op = {"done": False, "regions": regions}
        issued[who].append(op)
        reading.append(op)

        def fin():
            op["done"] = True
            reading.remove(op)
            done()
        async_op(fin)

    def busy(region):
        return any(region in op["regions"] for op in reading)

    def producer():
        def load(kind, t):
            st = kst if kind == "K" else vst
            nst = KS if kind == "K" else VS
            s = t % nst
            assert not busy((kind, s)), f"{kind} stage {s} reloaded while an MMA reads it"
            st[s] = None

            def ld(t=t, s=s):
                st[s] = t
                (kfull if kind == "K" else vfull)[s].arrive()
            async_op(ld)
        if n_tiles:
            load("K", 0)
            load("V", 0)
            yield (kfull[0], 0)
        for t in range(1, n_tiles):
            if t >= KS:
                yield (kfree[t % KS], ((t // KS) - 1) & 1)
            load("K", t)
            if t >= VS:
                yield (vfree[t % VS], ((t // VS) - 1) & 1)
            load("V", t)

    def s_issuer():
        for i in range(n_seq):
            g, k, t = seq(i)
            if not dual or g == 0:
                yield (kfull[t % KS], (t // KS) & 1)
            if k > 0:
                yield (pvdone[g], (k - 1) & 1)

            def chk(g=g, k=k, t=t):
                assert kst[t % KS] == t, f"S reads a K stage not holding tile {t}"
                assert pv_inflight[g] == 0 or s_buf[g] is None, "S overwrites P still read by a P.V"
                assert not holding[g], f"S overwrites slot {g}'s S that a softmax warp still reads"
                s_buf[g] = None

            def fin(g=g, t=t):
                s_buf[g] = t
                p_half[g].clear()
            mma("S", [("K", t % KS), ("S", g)], chk, fin)
            commit("S", sfull[g])
            if not dual or g == 1:
                commit("S", kfree[t % KS])
        commit("S", drain_s)
        yield (drain_s, 0)

    def pv_issuer():
        for i in range(n_seq):
            g, k, t = seq(i)
            if not dual or g == 0:
                yield (vfull[t % VS], (t // VS) & 1)
            for hh in range(2):
                yield ((phi if hh else plo)[g], k & 1)

                def chk(g=g, t=t, hh=hh):
                    assert s_buf[g] == t and hh in p_half[g], f"P.V reads P({g}, {t}) half {hh} not written"
                    assert vst[t % VS] == t, f"P.V reads a V stage not holding tile {t}"
                    pv_inflight[g] += 1

                def fin(g=g):
                    pv_inflight[g] -= 1
                mma("PV", [("V", t % VS), ("P", g)], chk, fin)
                if hh == 0:
                    commit("PV", pvlo[g])
            commit("PV", pvdone[g])
            if not dual or g == 1:
                commit("PV", vfree[t % VS])
        commit("PV", drain_pv)
        yield (drain_pv, 0)

    staged = []

    def softmax(g, w, barrier):
        for k in range(n_slot[g]):
            t = k if dual else 2 * k + g
            yield (sfull[g], k & 1)
            assert s_buf[g] == t, f"softmax reads S({g}, {t}) before it is done"
            holding[g].add(w)
            for hh in range(2):
                for _ in range(rnd.randint(0, 2)):
                    yield None
                if rnd.random() < lazy_prob and (k > 0 or hh == 1):
                    # rescale O: after the slot's previous P.V (first half) or this tile's
                    # first-half P.V (second half)
                    yield (pvlo[g], k & 1) if hh else (pvdone[g], (k - 1) & 1)
                    assert pv_inflight[g] == 0, "O rescaled while a P.V into it is in flight"
                if w == 0:
                    p_half[g].add(hh)
                if hh == 1:
                    holding[g].discard(w)
                (phi if hh else plo)[g].arrive()
        # epilogue
        if n_slot[g]:
            yield (pvdone[g], (n_slot[g] - 1) & 1)
        if dual and g == 0 and not stage_without_drain:
            yield (drain_s, 0)
        if dual:
            region = "K" if g == 0 else "V"
            for s in range(KS if region == "K" else VS):
                assert not busy((region, s)), f"slot {g} stages O into {region} stage {s} an MMA still reads"
                assert (kst if region == "K" else vst)[s] is not None, f"{region} stage {s} still loading"
        else:
            barrier[0] += 1
            while barrier[0] < 2 * n_warps:
                yield None
            for s in range(KS):
                assert not busy(("K", s)), f"O staged into K stage {s} an MMA still reads"
        staged.append((g, w))

    barrier = [0]
    actors = [producer(), s_issuer(), pv_issuer()] + [softmax(g, w, barrier) for g in range(2) for w in range(n_warps)]
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
            raise AssertionError(f"deadlock at n_tiles={n_tiles} dual={dual}")
    return True


@pytest.mark.parametrize("dual", [True, False])
@pytest.mark.parametrize("n_tiles", range(1, 10))
def test_dual_kernel_barrier_protocol(n_tiles, dual):
    for seed in range(60):
        assert run(n_tiles, dual, seed * 131 + n_tiles)


def test_model_finds_staging_before_the_last_s_mma():
    """Slot 0 of two row groups staging its O rows in the K stages without waiting for the S
    issuer's drain races with slot 1's last S MMA; the model must see it."""
    fails = 0
    for n_tiles in range(1, 8):
        for seed in range(60):
            try:
                run(n_tiles, True, seed * 7 + n_tiles, stage_without_drain=True)
            except AssertionError as e:
                assert "stages O into K stage" in str(e)
                fails += 1
    assert fails > 0
