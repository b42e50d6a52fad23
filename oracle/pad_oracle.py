"""fp64 CPU oracle for one event-factorized parallel decode step.

TEST INFRASTRUCTURE ONLY.  This module is the slow, obviously correct
definition that the CUDA path is checked against.  Only the test suite,
``__graft_entry__.smoke()`` and the CPU-baseline / reference arm of
``bench.py`` may import it; the product path (the ``paper_2607_02963_gb300``
package and its CUDA library) never does, and shares no code with it.

What it computes (Sec. 3.4 of the paper, Eq. 3 and the restructured causal
mask of Fig. 3): at decode step j every event branch i emits one token L^i_j at
once.  The query of branch i may attend to (1) the shared multimodal prefix P
together with all global event tokens G^1..G^K (the planning tokens live at the
end of the shared prefix), and (2) the tokens of its own branch (its anchor and
L^i_<j, plus the token appended at this step); tokens of any other branch are
masked out.  With one branch this is the ordinary causal decode of Eq. 1.

The method's result is exactly a masked softmax attention, so the oracle is
that plain definition written out: build each video's full key list, build the
explicit 0/1 event mask, and run a naive softmax in fp64.  Pinned by
``tests/test_oracle_pins.py`` (E=1 reduction and per-event reduction against
torch SDPA, permutation, perturbation, row sums, brute force, closed forms,
the log-sum-exp merge identity, and a hand-worked example under
``tests/golden/``).

Readings where the paper is silent (each also listed in the design notes):
  * the private length L_e given for a step excludes the token appended at
    this step, so branch e attends to L_e + 1 private keys;
  * the query head j of a GQA layer reads kv-head floor(j / G), G = H_q / H_kv;
  * scores are scale * q.k with scale = 1/sqrt(D); the LSE is natural-log;
  * new pages go to events in ascending event order, each taking the
    lowest-numbered free page; running out of pages changes nothing.
"""
from __future__ import annotations

import numpy as np


# ---------------------------------------------------------------------------
# bf16 -> fp64 (exact widening of the bit pattern)
# ---------------------------------------------------------------------------

def bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    """bf16 bit patterns (uint16) -> float64, exactly."""
    b = np.ascontiguousarray(bits, dtype=np.uint16)
    return (b.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)


# ---------------------------------------------------------------------------
# The explicit event-factorized mask (Sec. 3.4, Fig. 3)
# ---------------------------------------------------------------------------

def event_mask(prefix_len: int, branch_lens, self_g=None) -> np.ndarray:
    """Mask M[e, k] over the key sequence [prefix ; branch 1 ; ... ; branch E].

    M[e, k] is True when key k lies in the shared prefix (P and the planning
    tokens) or inside branch e's own block; keys of every other branch are
    False.  ``branch_lens[e]`` counts branch e's keys at this step (L_e + 1).

    ``self_g = (K, g_index)`` selects the "self G-token only" structure of the
    attention ablation (Tab. 8): the prefix ends with the planning tokens
    G^1..G^K and S (Sec. 3.3), and event e sees only G^(g_index[e] + 1) of them,
    besides P, S and its own branch.
    """
    branch_lens = [int(x) for x in branch_lens]
    n_keys = prefix_len + sum(branch_lens)
    M = np.zeros((len(branch_lens), n_keys), dtype=bool)
    M[:, :prefix_len] = True
    if self_g is not None:
        K, g_index = int(self_g[0]), [int(x) for x in self_g[1]]
        g0 = prefix_len - 1 - K                      # G^1 .. G^K, then S at prefix_len - 1
        for e in range(len(branch_lens)):
            M[e, g0:g0 + K] = False
            M[e, g0 + g_index[e]] = True
    start = prefix_len
    for e, n in enumerate(branch_lens):
        M[e, start:start + n] = True
        start += n
    return M


# ---------------------------------------------------------------------------
# Masked softmax attention for one video (all its events at once)
# ---------------------------------------------------------------------------

def video_attention(q, k_prefix, v_prefix, k_branches, v_branches, scale, return_p=False,
                    heads=None, self_g=None):
    """Decode attention of one video's events under the event-factorized mask.

    q:          [E_b, H_q, D] float64, one query token per event branch
    k_prefix:   [S, H_kv, D] float64 shared keys (prefix P + planning tokens)
    v_prefix:   [S, H_kv, D]
    k_branches: list of E_b arrays [n_e, H_kv, D] (branch e's keys, incl. this step's)
    v_branches: list of E_b arrays [n_e, H_kv, D]
    Returns o [E_b, H_q, D], lse [E_b, H_q] (natural log) and, when asked,
    the probabilities p [E_b, H_q, n_keys] over the full key sequence.
    ``heads`` restricts the work to those q-heads (the others are left at 0).
    """
    E_b, H_q, D = q.shape
    S, H_kv, _ = k_prefix.shape
    G = H_q // H_kv
    K_all = np.concatenate([k_prefix] + list(k_branches), axis=0)   # [n_keys, H_kv, D]
    V_all = np.concatenate([v_prefix] + list(v_branches), axis=0)
    M = event_mask(S, [kb.shape[0] for kb in k_branches], self_g)     # [E_b, n_keys]
    n_keys = K_all.shape[0]
    o = np.zeros((E_b, H_q, D), dtype=np.float64)
    lse = np.zeros((E_b, H_q), dtype=np.float64)
    p_all = np.zeros((E_b, H_q, n_keys), dtype=np.float64) if return_p else None
    for j in (range(H_q) if heads is None else heads):
        h = j // G                                   # contiguous GQA head mapping
        s = scale * (q[:, j, :] @ K_all[:, h, :].T)  # [E_b, n_keys]
        s = np.where(M, s, -np.inf)
        m = s.max(axis=1, keepdims=True)
        w = np.exp(s - m)                            # exp(-inf) = 0 for masked keys
        den = w.sum(axis=1, keepdims=True)
        p = w / den
        o[:, j, :] = p @ V_all[:, h, :]
        lse[:, j] = m[:, 0] + np.log(den[:, 0])
        if return_p:
            p_all[:, j, :] = p
    return o, lse, p_all


def decode_step(w, return_p=False, self_g=None):
    """Oracle for a whole batch described by a workload object (see ``synth.Workload``).

    Branch e's keys after this step's append are its L_e stored private tokens
    followed by k_new[e] (and likewise for values).  Returns o [E, H_q, D] and
    lse [E, H_q] in float64 (and p per video when asked).  ``self_g`` = (K per
    video, G index per event) selects the "self G-token only" mask (event_mask).
    """
    E = w.n_events
    o = np.zeros((E, w.h_q, w.head_dim), dtype=np.float64)
    lse = np.zeros((E, w.h_q), dtype=np.float64)
    ps = []
    for b in range(w.n_videos):
        ev = w.events_of_video(b)
        if ev.size == 0:
            continue
        qb = bf16_to_f64(w.q[ev])
        kp = bf16_to_f64(w.prefix_k(b))
        vp = bf16_to_f64(w.prefix_v(b))
        kbs = [np.concatenate([bf16_to_f64(w.priv_k(e)), bf16_to_f64(w.k_new[e:e + 1])]) for e in ev]
        vbs = [np.concatenate([bf16_to_f64(w.priv_v(e)), bf16_to_f64(w.v_new[e:e + 1])]) for e in ev]
        sg = None if self_g is None else (self_g[0][b], [self_g[1][e] for e in ev])
        ob, lb, pb = video_attention(qb, kp, vp, kbs, vbs, w.scale, return_p=return_p, self_g=sg)
        o[ev] = ob
        lse[ev] = lb
        ps.append(pb)
    if return_p:
        return o, lse, ps
    return o, lse


def event_rows(w, e, heads=None, self_g=None):
    """Oracle output of event e alone (all or selected q-heads), for sampled checks
    at full size: the mask of Sec. 3.4 restricted to row e is prefix + own branch."""
    b = int(w.event_video[e])
    qb = bf16_to_f64(w.q[e:e + 1])
    kp = bf16_to_f64(w.prefix_k(b))
    vp = bf16_to_f64(w.prefix_v(b))
    kb = np.concatenate([bf16_to_f64(w.priv_k(e)), bf16_to_f64(w.k_new[e:e + 1])])
    vb = np.concatenate([bf16_to_f64(w.priv_v(e)), bf16_to_f64(w.v_new[e:e + 1])])
    sg = None if self_g is None else (self_g[0][b], [self_g[1][e]])
    o, lse, _ = video_attention(qb, kp, vp, [kb], [vb], w.scale, heads=heads, self_g=sg)
    if heads is not None:
        return o[0, heads], lse[0, heads]
    return o[0], lse[0]


# ---------------------------------------------------------------------------
# Rotary position embedding at the shared per-step position (Sec. 3.4)
# ---------------------------------------------------------------------------
#
# Sec. 3.4 gives the tokens generated at the same decoding step of different
# branches identical position indices.  Positions enter attention through the
# rotary embedding of q and of the new key (values are not rotated); the prefix
# and earlier branch keys were rotated when they were written.  Reading (listed in
# the design notes): the rotate-half form over the whole head dimension, with a
# per-position table whose first D/2 columns hold cos(theta_i) and last D/2
# columns sin(theta_i); for the caption tokens of the paper's backbone all
# multimodal position components coincide, so this is the 1-D form.


def bf16_round(x32: np.ndarray) -> np.ndarray:
    """float32 values -> bf16 bit patterns (uint16), round to nearest, ties to even.

    Finite inputs only (the rotated values of finite bf16 rows and a finite table)."""
    u = np.ascontiguousarray(x32, dtype=np.float32).view(np.uint32).astype(np.uint64)
    lsb = (u >> np.uint64(16)) & np.uint64(1)
    return ((u + np.uint64(0x7FFF) + lsb) >> np.uint64(16)).astype(np.uint16)


def rope_rotate(x: np.ndarray, cs_row: np.ndarray) -> np.ndarray:
    """Rotate the rows x[..., D] by the table row cs_row[D] (cos | sin halves).

    Pairs (i, i + D/2): x'_i = x_i cos_i - x_{i+D/2} sin_i and
    x'_{i+D/2} = x_{i+D/2} cos_i + x_i sin_i.  Works in the dtype of its inputs:
    float64 for the exact rotation; float32 for the rounding of an unfused pass
    (each product and each sum rounded to float32, no fused multiply-add).
    """
    D = x.shape[-1]
    h = D // 2
    c, s = cs_row[:h], cs_row[h:]
    lo, hi = x[..., :h], x[..., h:]
    out = np.empty_like(x)
    out[..., :h] = lo * c - hi * s
    out[..., h:] = hi * c + lo * s
    return out


def rope_bits(bits: np.ndarray, cs_row32: np.ndarray) -> np.ndarray:
    """bf16 rows -> their rotation, as bf16 bits: widened exactly to float32,
    rotated in float32 (rope_rotate), rounded once to bf16."""
    x32 = bf16_to_f64(bits).astype(np.float32)
    return bf16_round(rope_rotate(x32, np.asarray(cs_row32, dtype=np.float32)))


def rotated_workload(w, positions, cos_sin32):
    """The workload with q and k_new rotated at each event's position (what an
    unfused RoPE pass would hand to attention and to the append)."""
    import dataclasses
    q = np.array(w.q, copy=True)
    kn = np.array(w.k_new, copy=True)
    for e in range(w.n_events):
        row = cos_sin32[int(positions[e])]
        q[e] = rope_bits(w.q[e], row)
        kn[e] = rope_bits(w.k_new[e], row)
    return dataclasses.replace(w, q=q, k_new=kn)


# ---------------------------------------------------------------------------
# Log-sum-exp merge of partial softmax states (the split-KV identity)
# ---------------------------------------------------------------------------

def lse_merge(parts):
    """Merge partial attention results over disjoint key sets.

    ``parts`` is a list of (o_s, lse_s) with o_s normalised over its own keys.
    The full result is o = sum_s exp(lse_s - LSE) o_s with LSE = log sum_s exp(lse_s).
    Parts with lse = -inf (no keys) contribute nothing.
    """
    lses = np.stack([np.asarray(l, dtype=np.float64) for _, l in parts])
    M = lses.max(axis=0)
    wts = np.exp(lses - M)
    tot = wts.sum(axis=0)
    o = sum(wts[s][..., None] * np.asarray(parts[s][0], dtype=np.float64)
            for s in range(len(parts))) / tot[..., None]
    return o, M + np.log(tot)


# ---------------------------------------------------------------------------
# Page bookkeeping of the fused append (one new token per branch per step)
# ---------------------------------------------------------------------------

OK = "ok"
OUT_OF_PAGES = "out_of_pages"
INVALID = "invalid"


def simulate_append(page_table, free_pages, event_len, page_size):
    """Where each branch's new token goes, and which pages get allocated.

    Walk the events in ascending order; an event whose pre-step length L_e is
    a multiple of the page size starts a new page and takes the lowest-numbered
    free page, recorded at page_table[e, L_e // page_size].  Its token goes to
    (page, L_e % page_size).  If the free pages do not cover every event that
    needs one, nothing changes.

    Returns (status, new_page_table, new_free_pages, slots[E, 2] = (page, offset)).
    """
    pt = np.array(page_table, dtype=np.int32, copy=True)
    free = sorted(int(x) for x in free_pages)
    L = [int(x) for x in event_len]
    E, max_pages = pt.shape if pt.ndim == 2 else (len(L), 0)
    if any(l < 0 or l // page_size >= max_pages for l in L):
        return INVALID, np.array(page_table, copy=True), np.array(sorted(free_pages)), None
    need = sum(1 for l in L if l % page_size == 0)
    if need > len(free):
        return OUT_OF_PAGES, np.array(page_table, copy=True), np.array(sorted(free_pages)), None
    slots = np.zeros((E, 2), dtype=np.int32)
    for e in range(E):
        idx = L[e] // page_size
        if L[e] % page_size == 0:
            pg = free.pop(0)
            pt[e, idx] = pg
        else:
            pg = int(pt[e, idx])
        slots[e] = (pg, L[e] % page_size)
    return OK, pt, np.array(free, dtype=np.int32), slots
