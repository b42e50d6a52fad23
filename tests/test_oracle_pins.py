"""Pins for the fp64 oracle: checks against what the paper and the mathematics fix.

None of these re-types the oracle's formula: they compare it with a library
routine (torch SDPA), a scalar brute force written separately, closed forms,
invariances that Eq. 3 implies, and hand-worked fixtures in tests/golden/.
"""
import json
import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle
from paper_2607_02963_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rand_video(rng, E, S, L, H_q=4, H_kv=2, D=16):
    q = rng.standard_normal((E, H_q, D))
    kp = rng.standard_normal((S, H_kv, D))
    vp = rng.standard_normal((S, H_kv, D))
    kb = [rng.standard_normal((n, H_kv, D)) for n in L]
    vb = [rng.standard_normal((n, H_kv, D)) for n in L]
    return q, kp, vp, kb, vb


def _sdpa_single(q_row, K, V, scale):
    """Library decode attention: one query [H_q, D] over keys K, V [n, H_kv, D] (GQA expanded
    with the contiguous mapping q-head j -> kv-head j // G)."""
    H_q = q_row.shape[0]
    H_kv = K.shape[1]
    G = H_q // H_kv
    qt = torch.from_numpy(q_row)[:, None, :]                                 # [H_q, 1, D]
    kt = torch.from_numpy(K).permute(1, 0, 2).repeat_interleave(G, dim=0)   # [H_q, n, D]
    vt = torch.from_numpy(V).permute(1, 0, 2).repeat_interleave(G, dim=0)
    out = F.scaled_dot_product_attention(qt, kt, vt, scale=scale)
    return out[:, 0, :].numpy()


# (i) E = 1 reduces to ordinary causal decode attention (Eq. 1).
@pytest.mark.parametrize("L", [0, 1, 7, 33])
def test_single_event_is_plain_decode(L):
    rng = np.random.default_rng(10 + L)
    q, kp, vp, kb, vb = _rand_video(rng, 1, 37, [L + 1])
    o, lse, _ = oracle.video_attention(q, kp, vp, kb, vb, 0.25)
    ref = _sdpa_single(q[0], np.concatenate([kp, kb[0]]), np.concatenate([vp, vb[0]]), 0.25)
    np.testing.assert_allclose(o[0], ref, rtol=1e-12, atol=1e-13)


# (ii) every event equals plain decode over concat(prefix, own branch) alone.
def test_each_event_is_decode_over_prefix_and_own_branch():
    rng = np.random.default_rng(3)
    L = [1, 4, 17, 9, 2]
    q, kp, vp, kb, vb = _rand_video(rng, len(L), 50, L, H_q=6, H_kv=2, D=8)
    o, _, _ = oracle.video_attention(q, kp, vp, kb, vb, 0.3)
    for e in range(len(L)):
        ref = _sdpa_single(q[e], np.concatenate([kp, kb[e]]), np.concatenate([vp, vb[e]]), 0.3)
        np.testing.assert_allclose(o[e], ref, rtol=1e-12, atol=1e-13)


# (iii) permuting the events permutes the outputs.
def test_permutation_equivariance():
    rng = np.random.default_rng(4)
    L = [3, 1, 6, 2]
    q, kp, vp, kb, vb = _rand_video(rng, 4, 21, L)
    o, lse, _ = oracle.video_attention(q, kp, vp, kb, vb, 0.5)
    perm = [2, 0, 3, 1]
    o2, lse2, _ = oracle.video_attention(q[perm], kp, vp, [kb[i] for i in perm],
                                         [vb[i] for i in perm], 0.5)
    np.testing.assert_allclose(o2, o[perm], rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(lse2, lse[perm], rtol=1e-13, atol=1e-14)


# (iv) an event's output ignores every other event's KV.
def test_other_events_kv_do_not_matter():
    rng = np.random.default_rng(5)
    L = [4, 2, 7]
    q, kp, vp, kb, vb = _rand_video(rng, 3, 19, L)
    o, lse, _ = oracle.video_attention(q, kp, vp, kb, vb, 0.5)
    kb2 = [kb[0]] + [100.0 * rng.standard_normal(x.shape) for x in kb[1:]]
    vb2 = [vb[0]] + [100.0 * rng.standard_normal(x.shape) for x in vb[1:]]
    o2, lse2, _ = oracle.video_attention(q, kp, vp, kb2, vb2, 0.5)
    assert np.array_equal(o2[0], o[0]) and np.array_equal(lse2[0], lse[0])
    # other branches of different length: same result up to summation order
    kb3 = [kb[0], rng.standard_normal((11, 2, 16)), rng.standard_normal((1, 2, 16))]
    vb3 = [vb[0], rng.standard_normal((11, 2, 16)), rng.standard_normal((1, 2, 16))]
    o3, _, _ = oracle.video_attention(q, kp, vp, kb3, vb3, 0.5)
    np.testing.assert_allclose(o3[0], o[0], rtol=1e-12, atol=1e-14)


# (v) softmax rows sum to one and put no weight on masked keys.
def test_rows_sum_to_one_and_mask_is_respected():
    rng = np.random.default_rng(6)
    L = [2, 5, 1]
    q, kp, vp, kb, vb = _rand_video(rng, 3, 13, L)
    _, _, p = oracle.video_attention(q, kp, vp, kb, vb, 1.0, return_p=True)
    np.testing.assert_allclose(p.sum(axis=-1), 1.0, rtol=0, atol=1e-12)
    starts = np.cumsum([13] + L)
    for e in range(3):
        for f in range(3):
            blk = p[e, :, starts[f]:starts[f] + L[f]]
            if f != e:
                assert np.all(blk == 0.0)
            else:
                assert np.all(blk > 0.0)


# (vi) a scalar brute force, written separately, agrees on tiny shapes.
def _brute(q, kp, vp, kb, vb, scale):
    E, H_q, D = q.shape
    H_kv = kp.shape[1]
    G = H_q // H_kv
    o = np.zeros_like(q)
    lse = np.zeros((E, H_q))
    for e in range(E):
        keys = [kp[t] for t in range(kp.shape[0])] + [kb[e][t] for t in range(kb[e].shape[0])]
        vals = [vp[t] for t in range(vp.shape[0])] + [vb[e][t] for t in range(vb[e].shape[0])]
        for j in range(H_q):
            h = j // G
            sc = []
            for key in keys:
                acc = 0.0
                for d in range(D):
                    acc += q[e, j, d] * key[h, d]
                sc.append(acc * scale)
            mx = max(sc)
            ws = [math.exp(x - mx) for x in sc]
            tot = sum(ws)
            for d in range(D):
                o[e, j, d] = sum(w * val[h, d] for w, val in zip(ws, vals)) / tot
            lse[e, j] = mx + math.log(tot)
    return o, lse


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_brute_force_tiny(seed):
    rng = np.random.default_rng(100 + seed)
    E = int(rng.integers(1, 4))
    L = [int(x) for x in rng.integers(1, 5, size=E)]
    S = int(rng.integers(0, 6))
    q, kp, vp, kb, vb = _rand_video(rng, E, S, L, H_q=4, H_kv=2, D=3)
    o, lse, _ = oracle.video_attention(q, kp, vp, kb, vb, 0.7)
    ob, lb = _brute(q, kp, vp, kb, vb, 0.7)
    np.testing.assert_allclose(o, ob, rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(lse, lb, rtol=1e-12, atol=1e-13)


# (vii) identical keys: uniform weights -> mean of the visible values; lse = s + ln(n).
def test_identical_keys_give_mean_of_visible_values():
    rng = np.random.default_rng(7)
    L = [3, 5]
    S = 9
    q, kp, vp, kb, vb = _rand_video(rng, 2, S, L, H_q=2, H_kv=1, D=4)
    key = rng.standard_normal(4)
    kp[:] = key
    for x in kb:
        x[:] = key
    o, lse, _ = oracle.video_attention(q, kp, vp, kb, vb, 0.5)
    for e in range(2):
        visible = np.concatenate([vp, vb[e]])[:, 0, :]
        np.testing.assert_allclose(o[e, 0], visible.mean(axis=0), rtol=1e-12, atol=1e-13)
        s = 0.5 * float(q[e, 0] @ key)
        np.testing.assert_allclose(lse[e, 0], s + math.log(S + L[e]), rtol=1e-12)


# (viii) constant values: the output is that constant whatever the weights.
def test_constant_values():
    rng = np.random.default_rng(8)
    L = [2, 6, 1]
    q, kp, vp, kb, vb = _rand_video(rng, 3, 11, L)
    c = rng.standard_normal(16)
    vp[:] = c
    for x in vb:
        x[:] = c
    o, _, _ = oracle.video_attention(q, kp, vp, kb, vb, 0.8)
    np.testing.assert_allclose(o, np.broadcast_to(c, o.shape), rtol=1e-12, atol=1e-13)


# lse pinned through a library routine: a zero key scores exactly 0, so its weight is
# exp(-lse); reading that weight out of SDPA with a one-hot value column gives -ln p_0.
def test_lse_against_sdpa_weight_of_zero_key():
    rng = np.random.default_rng(9)
    q, kp, vp, kb, vb = _rand_video(rng, 1, 12, [4], H_q=2, H_kv=1, D=6)
    kp[0] = 0.0
    vp[:, :, 0] = 0.0
    kb[0][:, :, 0] = 0.0
    vb[0][:, :, 0] = 0.0
    vp[0, :, 0] = 1.0
    _, lse, _ = oracle.video_attention(q, kp, vp, kb, vb, 0.6)
    ref = _sdpa_single(q[0], np.concatenate([kp, kb[0]]), np.concatenate([vp, vb[0]]), 0.6)
    np.testing.assert_allclose(lse[0], -np.log(ref[:, 0]), rtol=1e-12)


# (ix) the log-sum-exp merge of prefix-only and branch-only results equals the full result.
def test_lse_merge_identity():
    rng = np.random.default_rng(11)
    L = [5, 3]
    q, kp, vp, kb, vb = _rand_video(rng, 2, 30, L)
    o, lse, _ = oracle.video_attention(q, kp, vp, kb, vb, 0.4)
    empty = np.zeros((0, 2, 16))
    op, lp, _ = oracle.video_attention(q, kp, vp, [empty, empty], [empty, empty], 0.4)
    ob, lb, _ = oracle.video_attention(q, kp[:0], vp[:0], kb, vb, 0.4)
    # split the prefix further into three chunks
    parts = [(ob, lb)]
    for a, b in [(0, 7), (7, 19), (19, 30)]:
        parts.append(oracle.video_attention(q, kp[a:b], vp[a:b], [empty, empty], [empty, empty], 0.4)[:2])
    om, lm = oracle.lse_merge(parts)
    np.testing.assert_allclose(om, o, rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(lm, lse, rtol=1e-12, atol=1e-13)
    om2, lm2 = oracle.lse_merge([(op, lp), (ob, lb)])
    np.testing.assert_allclose(om2, o, rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(lm2, lse, rtol=1e-12, atol=1e-13)


def test_hand_worked_two_events():
    g = json.load(open(os.path.join(GOLDEN, "hand_two_events.json")))
    q = np.array(g["q"])
    kp = np.array(g["k_prefix"])
    vp = np.array(g["v_prefix"])
    kb = [np.array(x) for x in g["k_branches"]]
    vb = [np.array(x) for x in g["v_branches"]]
    o, lse, _ = oracle.video_attention(q, kp, vp, kb, vb, g["scale"])
    np.testing.assert_allclose(o, np.array(g["expect_o"]), rtol=1e-14)
    np.testing.assert_allclose(lse, np.array(g["expect_lse"]), rtol=1e-14)
    assert oracle.event_mask(2, [1, 1]).tolist() == g["expect_mask"]


def test_hand_worked_page_append():
    g = json.load(open(os.path.join(GOLDEN, "hand_page_append.json")))
    st, pt, free, slots = oracle.simulate_append(np.array(g["page_table"]), g["free_pages"],
                                                 g["event_len"], g["page_size"])
    assert st == oracle.OK
    assert pt.tolist() == g["expect_page_table"]
    assert free.tolist() == g["expect_free_pages"]
    assert slots.tolist() == g["expect_slots"]
    st, pt2, free2, slots = oracle.simulate_append(np.array(g["page_table"]),
                                                   g["out_of_pages_case"]["free_pages"],
                                                   g["event_len"], g["page_size"])
    assert st == g["out_of_pages_case"]["expect_status"] and slots is None
    assert pt2.tolist() == g["page_table"] and free2.tolist() == [0, 3]


def test_append_simulation_invariants():
    rng = np.random.default_rng(12)
    for trial in range(20):
        E = int(rng.integers(1, 12))
        ps = int(rng.choice([4, 16]))
        L = rng.integers(0, 50, size=E)
        maxp = int(L.max()) // ps + 2
        n_pages = 80
        perm = rng.permutation(n_pages)
        pt = np.full((E, maxp), -1, dtype=np.int32)
        cur = 0
        for e in range(E):
            for p in range((int(L[e]) + ps - 1) // ps):
                pt[e, p] = perm[cur]
                cur += 1
        free = np.sort(perm[cur:])
        st, pt2, free2, slots = oracle.simulate_append(pt, free, L, ps)
        assert st == oracle.OK
        need = [e for e in range(E) if L[e] % ps == 0]
        new = [int(pt2[e, L[e] // ps]) for e in need]
        assert new == sorted(new) and new == [int(x) for x in free[:len(need)]]
        assert sorted(free2.tolist() + new) == sorted(free.tolist())
        for e in range(E):
            assert slots[e, 0] == pt2[e, L[e] // ps] and slots[e, 1] == L[e] % ps


def test_decode_step_on_tiny_workload_matches_sdpa():
    """The whole-batch oracle on the tiny workload (bf16 inputs widened exactly) against SDPA."""
    w = synth.tiny()
    o, lse = oracle.decode_step(w)
    for e in range(w.n_events):
        K = np.concatenate([oracle.bf16_to_f64(w.prefix_k(0)), oracle.bf16_to_f64(w.priv_k(e)),
                            oracle.bf16_to_f64(w.k_new[e:e + 1])])
        V = np.concatenate([oracle.bf16_to_f64(w.prefix_v(0)), oracle.bf16_to_f64(w.priv_v(e)),
                            oracle.bf16_to_f64(w.v_new[e:e + 1])])
        ref = _sdpa_single(oracle.bf16_to_f64(w.q[e]), K, V, w.scale)
        np.testing.assert_allclose(o[e], ref, rtol=1e-11, atol=1e-12)


def test_bf16_widening_is_exact():
    x = np.array([1.0, -2.5, 3.140625, 0.0, -0.0], dtype=np.float32)
    bits = synth.f32_to_bf16_bits(x)
    np.testing.assert_array_equal(oracle.bf16_to_f64(bits), x.astype(np.float64))
    # round to nearest even at a tie: 1 + 2^-8 lies halfway between 1 and 1 + 2^-7
    tie = np.array([1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8], dtype=np.float32)
    np.testing.assert_array_equal(oracle.bf16_to_f64(synth.f32_to_bf16_bits(tie)),
                                  [1.0, 1.0 + 2.0 ** -6])


# ---------------------------------------------------------------------------
# Rotary embedding at the shared per-step position (Sec. 3.4)
# ---------------------------------------------------------------------------

def _exact_row(pos, D, theta=1.0e6):
    h = D // 2
    ang = pos * theta ** (-np.arange(h) * 2.0 / D)
    return np.concatenate([np.cos(ang), np.sin(ang)])


def test_bf16_round_matches_torch_and_ties_to_even():
    rng = np.random.default_rng(3)
    x = (rng.standard_normal(4096) * np.exp(rng.uniform(-20, 20, 4096))).astype(np.float32)
    want = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(oracle.bf16_round(x), want)
    # halfway between 1.0 (0x3F80) and the next bf16 up: ties to the even pattern
    assert oracle.bf16_round(np.array([1.0 + 2.0 ** -8], np.float32))[0] == 0x3F80
    assert oracle.bf16_round(np.array([1.0 + 3 * 2.0 ** -8], np.float32))[0] == 0x3F82


def test_rope_is_a_rotation_of_each_pair():
    """D = 2 closed form, and the norm of every (i, i + D/2) pair kept (fp64)."""
    th = 0.7
    x = np.array([[3.0, -2.0]])
    got = oracle.rope_rotate(x, np.array([math.cos(th), math.sin(th)]))
    want = np.array([[3 * math.cos(th) + 2 * math.sin(th), -2 * math.cos(th) + 3 * math.sin(th)]])
    assert np.allclose(got, want, rtol=0, atol=1e-15)
    rng = np.random.default_rng(4)
    D = 16
    x = rng.standard_normal((5, D))
    y = oracle.rope_rotate(x, _exact_row(1234, D))
    n0 = x[:, :D // 2] ** 2 + x[:, D // 2:] ** 2
    n1 = y[:, :D // 2] ** 2 + y[:, D // 2:] ** 2
    assert np.allclose(n0, n1, rtol=1e-13, atol=0)


def test_rope_scores_depend_on_relative_position_only():
    """<R(m) q, R(n) k> = <R(m+t) q, R(n+t) k> (fp64, exact tables), and rotations
    compose: R(b) R(a) x = R(a+b) x."""
    rng = np.random.default_rng(5)
    D = 32
    q, k = rng.standard_normal(D), rng.standard_normal(D)
    for m, n, t in [(10, 3, 7), (0, 500, 1234), (40000, 39000, 17)]:
        a = oracle.rope_rotate(q, _exact_row(m, D)) @ oracle.rope_rotate(k, _exact_row(n, D))
        b = oracle.rope_rotate(q, _exact_row(m + t, D)) @ oracle.rope_rotate(k, _exact_row(n + t, D))
        assert abs(a - b) <= 1e-9 * (1 + abs(a))
    x = rng.standard_normal(D)
    two = oracle.rope_rotate(oracle.rope_rotate(x, _exact_row(300, D)), _exact_row(77, D))
    assert np.allclose(two, oracle.rope_rotate(x, _exact_row(377, D)), rtol=0, atol=1e-12)


def test_rope_bits_identity_at_position_zero_and_float32_rounding():
    """Position 0 (cos 1, sin 0) gives back the input bits; elsewhere the float32
    rotation rounded once to bf16 is within one bf16 step of the exact rotation of the
    same (widened) inputs and table."""
    rng = np.random.default_rng(6)
    D = 128
    bits = synth.f32_to_bf16_bits(rng.standard_normal((7, D)).astype(np.float32))
    table = synth.rope_table(50000, D)
    assert np.array_equal(oracle.rope_bits(bits, table[0]), bits)
    for pos in (1, 8191, 32801, 49999):
        got = oracle.bf16_to_f64(oracle.rope_bits(bits, table[pos]))
        exact = oracle.rope_rotate(oracle.bf16_to_f64(bits), table[pos].astype(np.float64))
        step = np.maximum(np.abs(exact), 2.0 ** -126) * 2.0 ** -7
        assert np.all(np.abs(got - exact) <= step)


def test_rope_table_closed_form():
    t = synth.rope_table(40000, 128)
    for pos, i in [(0, 0), (1, 0), (1, 63), (32768, 5), (39999, 40)]:
        ang = pos * 1.0e6 ** (-2.0 * i / 128)
        assert t[pos, i] == np.float32(math.cos(ang))
        assert t[pos, 64 + i] == np.float32(math.sin(ang))


# ---------------------------------------------------------------------------
# "Self G-token only" mask variant (Tab. 8): G^1..G^K and S end the prefix
# ---------------------------------------------------------------------------

def _self_g_case(seed, E=3, S=20, K=4, D=16):
    rng = np.random.default_rng(seed)
    L = [int(x) for x in rng.integers(0, 5, size=E)]
    q, kp, vp, kbs, vbs = _rand_video(rng, E, S, L, D=D)
    g_index = [int(x) for x in rng.permutation(K)[:E]]
    return q, kp, vp, kbs, vbs, (K, g_index)


def test_self_g_mask_hides_exactly_the_other_events_g_tokens():
    E, S, K = 3, 20, 4
    M_full = oracle.event_mask(S, [2, 1, 3])
    M = oracle.event_mask(S, [2, 1, 3], (K, [2, 0, 3]))
    g0 = S - 1 - K
    for e, own in enumerate([2, 0, 3]):
        diff = np.nonzero(M_full[e] != M[e])[0]
        assert set(diff.tolist()) == {g0 + g for g in range(K) if g != own}
        assert M[e, S - 1] and M[e, :g0].all()        # S and P stay visible
    assert np.array_equal(oracle.event_mask(S, [2, 1, 3], (0, [0, 0, 0])), M_full)


def test_self_g_other_events_g_rows_do_not_matter():
    """Changing the K/V rows of G tokens an event cannot see leaves its output bit for
    bit; changing its own G row changes it."""
    q, kp, vp, kbs, vbs, sg = _self_g_case(8)
    scale = 1 / math.sqrt(q.shape[-1])
    K, g_index = sg
    o0, l0, _ = oracle.video_attention(q, kp, vp, kbs, vbs, scale, self_g=sg)
    S = kp.shape[0]
    g0 = S - 1 - K
    other = [g for g in range(K) if g != g_index[0]]
    kp2, vp2 = kp.copy(), vp.copy()
    kp2[g0 + other[0]] += 3.0
    vp2[g0 + other[1]] -= 2.0
    o1, l1, _ = oracle.video_attention(q, kp2, vp2, kbs, vbs, scale, self_g=sg)
    assert np.array_equal(o0[0], o1[0]) and np.array_equal(l0[0], l1[0])
    kp3 = kp.copy()
    kp3[g0 + g_index[0]] += 3.0
    o2, _, _ = oracle.video_attention(q, kp3, vp, kbs, vbs, scale, self_g=sg)
    assert not np.allclose(o0[0], o2[0])


def test_self_g_against_sdpa_on_the_visible_keys():
    """Event e's output equals plain attention over exactly P, its own G, S and its own
    branch (library routine on the gathered keys)."""
    q, kp, vp, kbs, vbs, sg = _self_g_case(9, E=2, S=30, K=5, D=8)
    scale = 1 / math.sqrt(q.shape[-1])
    K, g_index = sg
    o, _, _ = oracle.video_attention(q, kp, vp, kbs, vbs, scale, self_g=sg)
    S = kp.shape[0]
    g0 = S - 1 - K
    for e in range(q.shape[0]):
        rows = list(range(g0)) + [g0 + g_index[e], S - 1]
        Kv = np.concatenate([kp[rows], kbs[e]])
        Vv = np.concatenate([vp[rows], vbs[e]])
        assert np.allclose(o[e], _sdpa_single(q[e], Kv, Vv, scale), rtol=1e-10, atol=1e-12)


# ---------------------------------------------------------------------------
# "Causal attention" mask variant (Tab. 8): generated tokens of all branches visible
# ---------------------------------------------------------------------------

def test_causal_mask_shape():
    M = oracle.event_mask(5, [3, 1, 2], causal=True)
    want = np.zeros((3, 11), bool)
    want[:, :5] = True
    want[:, 5:7] = True      # branch 0's two stored tokens
    want[0, 7] = True        # its token of this step
    want[1, 8] = True        # branch 1 has no stored token
    want[:, 9:10] = True     # branch 2's stored token
    want[2, 10] = True
    assert np.array_equal(M, want)
    assert np.array_equal(oracle.event_mask(5, [4], causal=True), oracle.event_mask(5, [4]))


def test_causal_sees_stored_tokens_of_other_branches_but_not_their_new_one():
    rng = np.random.default_rng(11)
    q, kp, vp, kbs, vbs = _rand_video(rng, 3, 12, [4, 2, 5])
    scale = 0.3
    o0, _, _ = oracle.video_attention(q, kp, vp, kbs, vbs, scale, causal=True)
    k2 = [x.copy() for x in kbs]
    k2[1][-1] += 5.0                                # branch 1's token of this step
    o1, _, _ = oracle.video_attention(q, kp, vp, k2, vbs, scale, causal=True)
    assert np.array_equal(o0[0], o1[0]) and np.array_equal(o0[2], o1[2])
    assert not np.allclose(o0[1], o1[1])
    k3 = [x.copy() for x in kbs]
    k3[1][0] += 5.0                                 # a stored token of branch 1
    o2, _, _ = oracle.video_attention(q, kp, vp, k3, vbs, scale, causal=True)
    assert not np.allclose(o0[0], o2[0]) and not np.allclose(o0[2], o2[2])


def test_causal_against_sdpa_on_the_visible_keys():
    rng = np.random.default_rng(12)
    q, kp, vp, kbs, vbs = _rand_video(rng, 3, 9, [3, 1, 4], D=8)
    scale = 1 / math.sqrt(8)
    o, _, _ = oracle.video_attention(q, kp, vp, kbs, vbs, scale, causal=True)
    stored_k = np.concatenate([kb[:-1] for kb in kbs])
    stored_v = np.concatenate([vb[:-1] for vb in vbs])
    for e in range(3):
        Kv = np.concatenate([kp, stored_k, kbs[e][-1:]])
        Vv = np.concatenate([vp, stored_v, vbs[e][-1:]])
        assert np.allclose(o[e], _sdpa_single(q[e], Kv, Vv, scale), rtol=1e-10, atol=1e-12)


# ---------------------------------------------------------------------------
# Grounding readout (Sec. 3.3; inference by similarity matching)
# ---------------------------------------------------------------------------

def test_grounding_hand_worked_example():
    with open(os.path.join(os.path.dirname(__file__), "golden", "grounding_example.json")) as f:
        ex = json.load(f)
    sc = oracle.ground_segment_scores(ex["g_proj"], ex["f_proj"], ex["offsets"])
    assert np.allclose(sc, ex["scores"], rtol=0, atol=1e-15)
    for th in ("0.5", "0.7"):
        sal, iv = oracle.ground_salient(sc, float(th))
        assert np.array_equal(sal.astype(int), ex["threshold_" + th]["salient"])
        assert np.array_equal(iv, ex["threshold_" + th]["interval"])
    _, iv = oracle.ground_salient(sc, 0.5)
    out = oracle.attention_aggregate(ex["g_emb"], ex["f_proj"], ex["attn"], iv, ex["offsets"])
    assert np.allclose(out, ex["aggregate_at_0.5"], rtol=0, atol=1e-12)


def test_grounding_scores_brute_force():
    rng = np.random.default_rng(21)
    K, T, d = 3, 17, 5
    g, f = rng.standard_normal((K, d)), rng.standard_normal((T, d))
    offsets = [0, 4, 5, 11, 17]
    got = oracle.ground_segment_scores(g, f, offsets)
    for i in range(K):
        for s in range(4):
            tot = 0.0
            for t in range(offsets[s], offsets[s + 1]):
                for c in range(d):
                    tot += g[i, c] * f[t, c]
            assert abs(got[i, s] - tot) <= 1e-12


def test_grounding_threshold_rules():
    sc = np.array([[4.0, 2.0, 1.9, 4.0], [-3.0, -1.0, -2.0, -1.5]])
    sal, iv = oracle.ground_salient(sc, 0.5)
    assert sal[0].tolist() == [True, True, False, True] and iv[0].tolist() == [0, 3]
    assert sal[1].tolist() == [False, True, False, False] and iv[1].tolist() == [1, 1]  # no positive score
    rng = np.random.default_rng(22)
    sc = rng.standard_normal((6, 40)) + 1.0
    prev = None
    for th in (0.0, 0.3, 0.5, 0.7, 1.0):
        sal, _ = oracle.ground_salient(sc, th)
        assert sal[np.arange(6), sc.argmax(axis=1)].all()
        if prev is not None:
            assert not (sal & ~prev).any()                 # a higher fraction keeps a subset
        prev = sal


def test_attention_aggregate_special_cases():
    rng = np.random.default_rng(23)
    T, d, K = 12, 4, 2
    x, g = rng.standard_normal((T, d)), rng.standard_normal((K, d))
    offsets = [0, 3, 7, 12]
    iv = np.array([[0, 1], [2, 2]])
    uni = oracle.attention_aggregate(g, x, np.ones(T), iv, offsets)       # uniform: mean pooling
    assert np.allclose(uni[0], g[0] + x[0:7].mean(axis=0)) and np.allclose(uni[1], g[1] + x[7:12].mean(axis=0))
    hot = np.zeros(T)
    hot[5] = 0.7
    hot[9] = 0.2
    out = oracle.attention_aggregate(g, x, hot, iv, offsets)              # one weight in each range
    assert np.allclose(out[0], g[0] + x[5]) and np.allclose(out[1], g[1] + x[9])
    a = rng.uniform(0, 1, T)
    assert np.allclose(oracle.attention_aggregate(g, x, a, iv, offsets),
                       oracle.attention_aggregate(g, x, 3.5 * a, iv, offsets))  # weights normalised


# ---------------------------------------------------------------------------
# Full-sequence mask for training / prefill (Sec. 3.4, Fig. 3)
# ---------------------------------------------------------------------------

def test_prefill_mask_hand_worked():
    M = oracle.prefill_mask(3, [2, 1])
    want = np.array([[1, 0, 0, 0, 0, 0],
                     [1, 1, 0, 0, 0, 0],
                     [1, 1, 1, 0, 0, 0],
                     [1, 1, 1, 1, 0, 0],
                     [1, 1, 1, 1, 1, 0],
                     [1, 1, 1, 0, 0, 1]], dtype=bool)
    assert np.array_equal(M, want)


def test_prefill_without_branches_is_causal_attention():
    rng = np.random.default_rng(31)
    N, Hq, Hkv, D = 40, 4, 2, 16
    q, k, v = rng.standard_normal((N, Hq, D)), rng.standard_normal((N, Hkv, D)), rng.standard_normal((N, Hkv, D))
    o, _ = oracle.prefill_attention(q, k, v, N, [], 0.25)
    qt = torch.from_numpy(q).permute(1, 0, 2)
    kt = torch.from_numpy(k).permute(1, 0, 2).repeat_interleave(2, dim=0)
    vt = torch.from_numpy(v).permute(1, 0, 2).repeat_interleave(2, dim=0)
    ref = F.scaled_dot_product_attention(qt, kt, vt, is_causal=True, scale=0.25).permute(1, 0, 2).numpy()
    assert np.allclose(o, ref, rtol=1e-10, atol=1e-12)


def test_prefill_last_branch_token_is_the_decode_step():
    """The last token of each branch in the full-sequence mask is exactly that branch's
    decode step (the decode oracle over the prefix and the branch's tokens)."""
    rng = np.random.default_rng(32)
    S, lens, Hq, Hkv, D = 10, [3, 1, 4], 4, 2, 8
    N = S + sum(lens)
    q, k, v = rng.standard_normal((N, Hq, D)), rng.standard_normal((N, Hkv, D)), rng.standard_normal((N, Hkv, D))
    o, lse = oracle.prefill_attention(q, k, v, S, lens, 0.3)
    starts = np.cumsum([S] + lens[:-1])
    last = [int(st + n - 1) for st, n in zip(starts, lens)]
    kb = [k[st:st + n] for st, n in zip(starts, lens)]
    vb = [v[st:st + n] for st, n in zip(starts, lens)]
    od, ld, _ = oracle.video_attention(q[last], k[:S], v[:S], kb, vb, 0.3)
    assert np.allclose(o[last], od, rtol=1e-12, atol=1e-12) and np.allclose(lse[last], ld, rtol=1e-12, atol=1e-12)


def test_prefill_other_branches_do_not_matter():
    rng = np.random.default_rng(33)
    S, lens, Hq, Hkv, D = 6, [2, 3], 2, 1, 4
    N = S + sum(lens)
    q, k, v = rng.standard_normal((N, Hq, D)), rng.standard_normal((N, Hkv, D)), rng.standard_normal((N, Hkv, D))
    o0, _ = oracle.prefill_attention(q, k, v, S, lens, 0.5)
    k2, v2 = k.copy(), v.copy()
    k2[S + 2:] += 4.0                      # branch 2's tokens
    v2[S + 2:] -= 1.0
    o1, _ = oracle.prefill_attention(q, k2, v2, S, lens, 0.5)
    assert np.array_equal(o0[:S + 2], o1[:S + 2])   # prefix and branch 1 unchanged
    assert not np.allclose(o0[S + 2:], o1[S + 2:])


# ---------------------------------------------------------------------------
# event_rows, rotated_workload and decode_step on several videos
# ---------------------------------------------------------------------------
# The full-size GPU checks call event_rows (one event at a time) and the RoPE checks
# call rotated_workload, so both are pinned here against things fixed outside the
# oracle: keys gathered by hand from the raw workload arrays, the library's SDPA, and
# a hand-worked rotation table.

def _widen(bits):
    """bf16 bits -> float64 through torch's own bf16 type (independent of the oracle)."""
    t = torch.from_numpy(np.ascontiguousarray(bits, dtype=np.uint16).view(np.int16))
    return t.view(torch.bfloat16).double().numpy()


def _hand_keys(w, e, causal=False, self_g=None):
    """Event e's visible keys and values in decode order, gathered from the raw arrays.

    Plain mask: its video's prefix rows, its stored branch rows, its new row.  With
    ``causal``: the prefix, the stored rows of every branch of its video, its new row.
    With ``self_g = (K per video, G index per event)``: prefix rows outside the video's
    planning tokens, plus its own G token."""
    b = int(w.event_video[e])
    off, n = int(w.prefix_offset[b]), int(w.prefix_len[b])
    rows = list(range(off, off + n))
    if self_g is not None and int(self_g[0][b]) > 0:
        K = int(self_g[0][b])
        g0 = off + n - 1 - K
        rows = [r for r in rows if not (g0 <= r < g0 + K) or r == g0 + int(self_g[1][e])]
    ks, vs = [w.k_prefix[rows]], [w.v_prefix[rows]]
    owners = [f for f in range(w.n_events) if int(w.event_video[f]) == b] if causal else [e]
    for f in owners:
        ks.append(w.k_priv[int(w.priv_off[f]):int(w.priv_off[f + 1])])
        vs.append(w.v_priv[int(w.priv_off[f]):int(w.priv_off[f + 1])])
    ks.append(w.k_new[e:e + 1])
    vs.append(w.v_new[e:e + 1])
    return _widen(np.concatenate(ks)), _widen(np.concatenate(vs))


def _multi_video(seed):
    """A small ragged batch of at least two videos whose prefixes differ."""
    for s in range(seed, seed + 200):
        w = synth.random_small(s, h_q=6, h_kv=2, head_dim=16, max_videos=3, max_prefix=40,
                               max_events=4, max_len=9)
        if w.n_videos >= 2 and len(set(w.event_video.tolist())) >= 2:
            return w
    raise AssertionError("no multi-video workload drawn")


@pytest.mark.parametrize("seed", [31, 57])
def test_event_rows_match_the_step_and_sdpa_on_several_videos(seed):
    w = _multi_video(seed)
    o, lse = oracle.decode_step(w)
    for e in range(w.n_events):
        oe, le = oracle.event_rows(w, e)
        np.testing.assert_allclose(oe, o[e], rtol=1e-12, atol=1e-13)
        np.testing.assert_allclose(le, lse[e], rtol=1e-13, atol=1e-13)
        oh, lh = oracle.event_rows(w, e, heads=[1, 4])
        np.testing.assert_allclose(oh, o[e, [1, 4]], rtol=1e-12, atol=1e-13)
        np.testing.assert_allclose(lh, lse[e, [1, 4]], rtol=1e-13, atol=1e-13)
        K, V = _hand_keys(w, e)
        ref = _sdpa_single(_widen(w.q[e]), K, V, w.scale)
        np.testing.assert_allclose(oe, ref, rtol=1e-11, atol=1e-12)


def _rope_case():
    """D = 4, one kv-head, four events: q and k_new rows [1, 2, 3, 4] (and 5..8 for
    event 1), v_new rows distinct.  Table rows: 0 = identity; 1 = pair 0 turned by
    90 degrees, pair 1 by 180; 2 = pair 0 by 180, pair 1 by 90 (all exact in fp32)."""
    w = synth.make_workload("rope_d4", 5, 2, 1, 4, [6], [4], [0, 1, 2, 3])
    base = np.array([1.0, 2.0, 3.0, 4.0], np.float32)
    q = np.tile(base, (4, 2, 1))
    q[1] = np.array([5.0, 6.0, 7.0, 8.0], np.float32)
    kn = np.tile(base, (4, 1, 1))
    kn[1] = np.array([5.0, 6.0, 7.0, 8.0], np.float32)
    w.q = synth.f32_to_bf16_bits(q)
    w.k_new = synth.f32_to_bf16_bits(kn)
    table = np.array([[1, 1, 0, 0], [0, -1, 1, 0], [-1, 0, 0, 1]], np.float32)
    return w, table


def test_rotated_workload_hand_worked_d4():
    w, table = _rope_case()
    pos = np.array([1, 2, 0, 1], np.int32)
    r = oracle.rotated_workload(w, pos, table)
    # x' = (x0 c0 - x2 s0, x1 c1 - x3 s1, x2 c0 + x0 s0, x3 c1 + x1 s1), worked by hand:
    want_q = {0: [-3.0, -2.0, 1.0, -4.0],     # [1,2,3,4] at row 1
              1: [-5.0, -8.0, -7.0, 6.0],     # [5,6,7,8] at row 2
              2: [1.0, 2.0, 3.0, 4.0],        # row 0: unchanged
              3: [-3.0, -2.0, 1.0, -4.0]}     # same input, same position as event 0
    for e, row in want_q.items():
        assert np.array_equal(_widen(r.q[e]), np.array([row, row])), e
        assert np.array_equal(_widen(r.k_new[e]), np.array([row])), e
    # values, the prefix and the stored branch keys are never rotated
    for name in ("v_new", "k_prefix", "v_prefix", "k_priv", "v_priv", "page_table"):
        assert np.array_equal(getattr(r, name), getattr(w, name)), name
    # the caller's workload is left as it was
    assert np.array_equal(_widen(w.q[0, 0]), [1.0, 2.0, 3.0, 4.0])


def test_rotated_workload_uses_each_events_own_position():
    """Only the events whose position is not 0 change; two events with equal rows at
    the same position get the same rotation (Sec. 3.4: one position per step)."""
    rng = np.random.default_rng(8)
    w = synth.make_workload("rope_pos", 8, 4, 2, 16, [30], [5], [1, 0, 2, 3, 1], rng=rng)
    w.q[3] = w.q[1]
    w.k_new[3] = w.k_new[1]
    table = synth.rope_table(64, 16)
    for moved in range(w.n_events):
        pos = np.zeros(w.n_events, np.int32)
        pos[moved] = 37
        r = oracle.rotated_workload(w, pos, table)
        for e in range(w.n_events):
            same_q = np.array_equal(r.q[e], w.q[e])
            same_k = np.array_equal(r.k_new[e], w.k_new[e])
            assert same_q == same_k == (e != moved), (moved, e)
        assert np.array_equal(r.v_new, w.v_new)
    pos = np.array([5, 37, 9, 37, 2], np.int32)
    r = oracle.rotated_workload(w, pos, table)
    assert np.array_equal(r.q[1], r.q[3]) and np.array_equal(r.k_new[1], r.k_new[3])
    pos[3] = 38
    r2 = oracle.rotated_workload(w, pos, table)
    assert not np.array_equal(r2.q[1], r2.q[3])
    # each rotated row is within one bf16 step of the exact rotation of its own row
    for e in range(w.n_events):
        c, s = table[pos[e], :8].astype(np.float64), table[pos[e], 8:].astype(np.float64)
        x = _widen(w.k_new[e])
        exact = np.concatenate([x[..., :8] * c - x[..., 8:] * s, x[..., 8:] * c + x[..., :8] * s], -1)
        got = _widen(r2.k_new[e])
        assert np.all(np.abs(got - exact) <= np.maximum(np.abs(exact), 2.0 ** -126) * 2.0 ** -7)


@pytest.mark.parametrize("variant", ["self_g", "causal"])
def test_decode_step_variants_on_several_videos_against_sdpa(variant):
    """decode_step with the mask variants over a batch of videos: each event against the
    library's SDPA over the keys its video and the variant make visible, gathered by hand."""
    w = _multi_video(77)
    sg = None
    if variant == "self_g":
        Kp = np.array([min(int(w.prefix_len[b]) - 1, 3 + b) for b in range(w.n_videos)], np.int32)
        gi = np.zeros(w.n_events, np.int32)
        for b in range(w.n_videos):
            ev = w.events_of_video(b)
            if Kp[b] > 0:
                gi[ev] = (np.arange(len(ev)) * 2 + b) % Kp[b]
        sg = (Kp, gi)
    o, lse = oracle.decode_step(w, self_g=sg, causal=(variant == "causal"))
    for e in range(w.n_events):
        K, V = _hand_keys(w, e, causal=(variant == "causal"), self_g=sg)
        ref = _sdpa_single(_widen(w.q[e]), K, V, w.scale)
        np.testing.assert_allclose(o[e], ref, rtol=1e-11, atol=1e-12)
