"""Seeded synthetic workloads for one event-factorized decode step.

This module only draws and lays out inputs: lengths, bf16 query/key/value
tensors, and the pre-step page pool of each event's private KV.  It contains
none of the attention arithmetic, so both the fp64 oracle and the CUDA path
consume exactly the same arrays without sharing any computation.

Shapes follow the paper's decode setting (Sec. 3.4, Eq. 3): a batch of videos,
each with a shared prefix (audio-visual tokens plus the planning tokens
G^1..G^K and S, Sec. 3.3), and E_b event branches per video, each with its own
private tokens L^i_<j.  Every tensor is bf16 (round-to-nearest-even from fp32
N(0,1) samples) and is returned as raw uint16 bit patterns.

Draw order for a workload with seed s (numpy.random.default_rng(s)):
  1. lengths (prefix lengths, events per video, private lengths);
  2. Q, K_prefix, V_prefix, K_priv, V_priv, k_new, v_new, all N(0,1) float32;
  3. optional per-(kv-head, channel) LogNormal(0, sigma) scale, multiplied
     into every K (prefix, private and new) before the bf16 rounding;
  4. a random permutation of the page pool that places the private KV.
"""
from __future__ import annotations

import dataclasses
from typing import Optional, Sequence

import numpy as np

BF16_NAN = np.uint16(0x7FC0)


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 to bf16 (round to nearest, ties to even); return uint16 bits."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    if not np.all(np.isfinite(x)):
        raise ValueError("bf16 rounding expects finite inputs")
    u = x.view(np.uint32)
    r = (u + (np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1)))) >> np.uint32(16)
    return r.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float32 (used for device upload helpers)."""
    b = np.ascontiguousarray(b, dtype=np.uint16)
    return (b.astype(np.uint32) << np.uint32(16)).view(np.float32)


@dataclasses.dataclass
class Workload:
    """One decode step's inputs.  All bf16 tensors are uint16 bit patterns."""

    name: str
    seed: int
    h_q: int
    h_kv: int
    head_dim: int
    page_size: int
    scale: float
    prefix_len: np.ndarray      # [B] int32
    prefix_offset: np.ndarray   # [B] int64, token offset into k_prefix / v_prefix
    event_video: np.ndarray     # [E] int32, non-decreasing
    event_len: np.ndarray       # [E] int32, private length before this step
    q: np.ndarray               # [E, H_q, D]
    k_prefix: np.ndarray        # [T_tot, H_kv, D]
    v_prefix: np.ndarray        # [T_tot, H_kv, D]
    priv_off: np.ndarray        # [E+1] int64, offsets into k_priv / v_priv
    k_priv: np.ndarray          # [sum L_e, H_kv, D]
    v_priv: np.ndarray          # [sum L_e, H_kv, D]
    k_new: np.ndarray           # [E, H_kv, D]
    v_new: np.ndarray           # [E, H_kv, D]
    n_pages: int
    max_pages: int
    page_table: np.ndarray      # [E, max_pages] int32, -1 where unused (pre-step)
    free_pages: np.ndarray      # sorted int32 free page ids (pre-step)

    @property
    def n_videos(self) -> int:
        return int(self.prefix_len.shape[0])

    @property
    def n_events(self) -> int:
        return int(self.event_len.shape[0])

    @property
    def group(self) -> int:
        return self.h_q // self.h_kv

    def events_of_video(self, b: int) -> np.ndarray:
        return np.nonzero(self.event_video == b)[0]

    def priv_k(self, e: int) -> np.ndarray:
        return self.k_priv[self.priv_off[e]:self.priv_off[e + 1]]

    def priv_v(self, e: int) -> np.ndarray:
        return self.v_priv[self.priv_off[e]:self.priv_off[e + 1]]

    def prefix_k(self, b: int) -> np.ndarray:
        o = int(self.prefix_offset[b])
        return self.k_prefix[o:o + int(self.prefix_len[b])]

    def prefix_v(self, b: int) -> np.ndarray:
        o = int(self.prefix_offset[b])
        return self.v_prefix[o:o + int(self.prefix_len[b])]

    def build_pools(self, fill_nan: bool = True):
        """Pre-step page pools [n_pages, H_kv, page, D] holding each event's private KV.

        Slots that hold no valid token are filled with bf16 NaN (when
        ``fill_nan``), so a kernel that lets an invalid slot reach its result
        produces NaN instead of a plausible number.
        """
        ps, hk, d = self.page_size, self.h_kv, self.head_dim
        shape = (self.n_pages, hk, ps, d)
        fill = BF16_NAN if fill_nan else np.uint16(0)
        kp = np.full(shape, fill, dtype=np.uint16)
        vp = np.full(shape, fill, dtype=np.uint16)
        for e in range(self.n_events):
            k = self.priv_k(e)
            v = self.priv_v(e)
            for t in range(k.shape[0]):
                pg = self.page_table[e, t // ps]
                kp[pg, :, t % ps, :] = k[t]
                vp[pg, :, t % ps, :] = v[t]
        return kp, vp

    def bytes_algorithmic(self) -> dict:
        """Algorithmic HBM bytes of one step: prefix read once + branch KV + Q + out + append."""
        kv_tok = 2 * self.h_kv * self.head_dim * 2          # K and V, bf16
        prefix = int(self.prefix_len.sum()) * kv_tok
        branch = int((self.event_len + 1).sum()) * kv_tok
        q = self.n_events * self.h_q * self.head_dim * 2
        out = self.n_events * self.h_q * self.head_dim * 4 + self.n_events * self.h_q * 4
        append = self.n_events * kv_tok * 2                  # read k_new/v_new, write slots
        return dict(prefix=prefix, branch=branch, q=q, out=out, append=append,
                    total=prefix + branch + q + out + append)


def rope_table(max_position: int, head_dim: int, theta: float = 1.0e6) -> np.ndarray:
    """The rotary-embedding table a model keeps for its positions: fp32 [max_position,
    head_dim], cos(pos * theta^(-2i/D)) in columns i < D/2 and the matching sin in columns
    D/2 + i (computed in fp64, rounded once).  theta = 1e6 as in the paper's backbone
    family; an input of the step, like the weights that produce q and k."""
    h = head_dim // 2
    inv = theta ** (-np.arange(h, dtype=np.float64) * 2.0 / head_dim)
    ang = np.arange(max_position, dtype=np.float64)[:, None] * inv[None, :]
    return np.concatenate([np.cos(ang), np.sin(ang)], axis=1).astype(np.float32)


def step_positions(w) -> np.ndarray:
    """Per-event position of this step's token: the video's prefix length plus the
    branch's private length before the step, so branches at the same step share it
    (Sec. 3.4).  int32 [n_events]."""
    return (w.prefix_len[w.event_video].astype(np.int64) + w.event_len).astype(np.int32)


def _normal(rng, shape):
    return rng.standard_normal(size=shape, dtype=np.float32)


def make_workload(name: str, seed: int, h_q: int, h_kv: int, head_dim: int,
                  prefix_len: Sequence[int], events_per_video: Sequence[int],
                  event_len: Sequence[int], rng: Optional[np.random.Generator] = None,
                  k_scale_sigma: Optional[float] = None, page_size: int = 16,
                  spare_pages: Optional[int] = None, scale: Optional[float] = None) -> Workload:
    """Draw tensors for given lengths (lengths must already be drawn from ``rng``)."""
    if rng is None:
        rng = np.random.default_rng(seed)
    prefix_len = np.asarray(prefix_len, dtype=np.int32)
    epv = np.asarray(events_per_video, dtype=np.int32)
    event_len = np.asarray(event_len, dtype=np.int32)
    B = prefix_len.shape[0]
    assert epv.shape[0] == B and int(epv.sum()) == event_len.shape[0]
    E = int(event_len.shape[0])
    event_video = np.repeat(np.arange(B, dtype=np.int32), epv)
    prefix_offset = np.zeros(B, dtype=np.int64)
    if B > 1:
        prefix_offset[1:] = np.cumsum(prefix_len[:-1], dtype=np.int64)
    T = int(prefix_len.sum())
    priv_off = np.zeros(E + 1, dtype=np.int64)
    priv_off[1:] = np.cumsum(event_len, dtype=np.int64)
    NL = int(priv_off[-1])
    D = head_dim

    q = _normal(rng, (E, h_q, D))
    kpre = _normal(rng, (T, h_kv, D))
    vpre = _normal(rng, (T, h_kv, D))
    kpriv = _normal(rng, (NL, h_kv, D))
    vpriv = _normal(rng, (NL, h_kv, D))
    knew = _normal(rng, (E, h_kv, D))
    vnew = _normal(rng, (E, h_kv, D))
    if k_scale_sigma is not None:
        ks = rng.lognormal(0.0, k_scale_sigma, size=(h_kv, D)).astype(np.float32)
        kpre *= ks
        kpriv *= ks
        knew *= ks

    ps = page_size
    pages_used = [(int(l) + ps - 1) // ps for l in event_len]
    n_new = int(sum(1 for l in event_len if int(l) % ps == 0))
    if spare_pages is None:
        spare_pages = max(8, E // 2)
    n_pages = int(sum(pages_used)) + n_new + spare_pages
    max_pages = max(1, (int(event_len.max(initial=0)) + 1 + ps - 1) // ps + 1)
    perm = rng.permutation(n_pages).astype(np.int32)
    page_table = np.full((E, max_pages), -1, dtype=np.int32)
    cur = 0
    for e in range(E):
        for p in range(pages_used[e]):
            page_table[e, p] = perm[cur]
            cur += 1
    free_pages = np.sort(perm[cur:]).astype(np.int32)

    if scale is None:
        scale = 1.0 / float(np.sqrt(D))
    return Workload(
        name=name, seed=seed, h_q=h_q, h_kv=h_kv, head_dim=D, page_size=ps, scale=float(scale),
        prefix_len=prefix_len, prefix_offset=prefix_offset, event_video=event_video,
        event_len=event_len, q=f32_to_bf16_bits(q), k_prefix=f32_to_bf16_bits(kpre),
        v_prefix=f32_to_bf16_bits(vpre), priv_off=priv_off, k_priv=f32_to_bf16_bits(kpriv),
        v_priv=f32_to_bf16_bits(vpriv), k_new=f32_to_bf16_bits(knew), v_new=f32_to_bf16_bits(vnew),
        n_pages=n_pages, max_pages=max_pages, page_table=page_table, free_pages=free_pages)


# ---------------------------------------------------------------------------
# The five workloads (tiny, 8k, long 32k, ragged serving batch, event sweep).
# "uniform in [a, b]" means integers inclusive of both ends.
# ---------------------------------------------------------------------------

def tiny(seed: int = 1) -> Workload:
    """batch 1, H_q=4, H_kv=1, D=64; prefix 512 (496 audio-visual + 16 planning); E=4, L={0,5,11,16}."""
    rng = np.random.default_rng(seed)
    return make_workload("tiny_h4_d64_p512_e4", seed, 4, 1, 64, [512], [4], [0, 5, 11, 16], rng=rng)


def gqa_8k(seed: int = 2) -> Workload:
    """batch 1, H_q=28, H_kv=4, D=128; prefix 8192 (8176 + 16 planning); E=8, L uniform in [0, 64]."""
    rng = np.random.default_rng(seed)
    L = rng.integers(0, 64 + 1, size=8)
    return make_workload("gqa_h28_d128_p8192_e8", seed, 28, 4, 128, [8192], [8], L, rng=rng)


def long_32k(seed: int = 3) -> Workload:
    """batch 1, H_q=28, H_kv=4, D=128; prefix 32768 (32736 + 32 planning); E=32, L uniform in [0, 128];
    K per-channel scale LogNormal(0, 0.5) to mimic outlier channels."""
    rng = np.random.default_rng(seed)
    L = rng.integers(0, 128 + 1, size=32)
    return make_workload("long_h28_d128_p32768_e32", seed, 28, 4, 128, [32768], [32], L, rng=rng,
                         k_scale_sigma=0.5)


def ragged_serving(seed: int = 4) -> Workload:
    """16 videos, H_q=28, H_kv=4, D=128; prefix uniform in [4096, 16384] + 16 planning tokens;
    E per video uniform in [4, 24]; private lengths uniform in [0, 96]."""
    rng = np.random.default_rng(seed)
    P = rng.integers(4096, 16384 + 1, size=16) + 16
    Ev = rng.integers(4, 24 + 1, size=16)
    L = rng.integers(0, 96 + 1, size=int(Ev.sum()))
    return make_workload("ragged_b16_h28_d128", seed, 28, 4, 128, P, Ev, L, rng=rng)


def event_sweep(E: int, seed: Optional[int] = None) -> Workload:
    """batch 1, H_q=28, H_kv=4, D=128; prefix 16384; E events with private length fixed at 48."""
    if seed is None:
        seed = 100 + E
    rng = np.random.default_rng(seed)
    return make_workload(f"sweep_h28_d128_p16384_e{E}", seed, 28, 4, 128, [16384], [E], [48] * E,
                         rng=rng)


SWEEP_E = (1, 2, 4, 8, 16, 32, 64)


def random_small(seed: int, h_q: int = 8, h_kv: int = 2, head_dim: int = 128,
                 max_videos: int = 3, max_prefix: int = 700, max_events: int = 6,
                 max_len: int = 40, k_scale_sigma: Optional[float] = None) -> Workload:
    """Small random ragged workload for parity sweeps (several tiles plus a ragged tail)."""
    rng = np.random.default_rng(seed)
    B = int(rng.integers(1, max_videos + 1))
    P = rng.integers(1, max_prefix + 1, size=B)
    Ev = rng.integers(1, max_events + 1, size=B)
    L = rng.integers(0, max_len + 1, size=int(Ev.sum()))
    return make_workload(f"small_s{seed}", seed, h_q, h_kv, head_dim, P, Ev, L, rng=rng,
                         k_scale_sigma=k_scale_sigma)


@dataclasses.dataclass
class GroundingInputs:
    """Seeded stand-ins for the grounding readout of one video (Sec. 3.3): projected
    audio-visual prefix tokens and event tokens, the segment ranges, the prefix hidden
    states, the last query token's attention on the prefix, and the event embeddings."""
    offsets: np.ndarray    # [S + 1] int32, token ranges of the time segments
    f_proj: np.ndarray     # [T, d_proj] bf16 bits
    g_proj: np.ndarray     # [K, d_proj] bf16 bits
    x: np.ndarray          # [T, d_model] bf16 bits
    attn: np.ndarray       # [T] fp32, non-negative, sums to 1 over the prefix
    g_emb: np.ndarray      # [K, d_model] bf16 bits
    true_seg: np.ndarray   # [K, 2] the segment range each event token was drawn near


def grounding_inputs(seed: int, n_tokens: int, n_segments: int, n_events: int, d_proj: int,
                     d_model: int, text_tokens: int = 0) -> GroundingInputs:
    """Segments of near-equal length after `text_tokens` leading text tokens; each event
    token is the mean projected feature of a random run of 1-4 segments plus noise, so it
    has a real best interval; attention weights are a softmax of N(0, 1) logits."""
    rng = np.random.default_rng(seed)
    av = n_tokens - text_tokens
    cuts = np.sort(rng.choice(np.arange(1, av), size=n_segments - 1, replace=False)) if n_segments > 1 else []
    offsets = (text_tokens + np.concatenate([[0], cuts, [av]])).astype(np.int32)
    f = _normal(rng, (n_tokens, d_proj))
    seg_mean = np.stack([f[offsets[s]:offsets[s + 1]].mean(axis=0) for s in range(n_segments)])
    true = np.zeros((n_events, 2), dtype=np.int32)
    g = np.zeros((n_events, d_proj), dtype=np.float32)
    for i in range(n_events):
        w = int(rng.integers(1, 5))
        s0 = int(rng.integers(0, max(1, n_segments - w + 1)))
        true[i] = (s0, min(n_segments, s0 + w) - 1)
        g[i] = 8.0 * seg_mean[s0:s0 + w].mean(axis=0) + 0.1 * _normal(rng, (d_proj,))
    x = _normal(rng, (n_tokens, d_model))
    logits = _normal(rng, (n_tokens,)).astype(np.float64)
    a = np.exp(logits - logits.max())
    a = (a / a.sum()).astype(np.float32)
    emb = _normal(rng, (n_events, d_model))
    return GroundingInputs(offsets=offsets, f_proj=f32_to_bf16_bits(f), g_proj=f32_to_bf16_bits(g),
                           x=f32_to_bf16_bits(x), attn=a, g_emb=f32_to_bf16_bits(emb), true_seg=true)


def prefill_inputs(seed: int, prefix_len: int, branch_lens, h_q: int, h_kv: int, head_dim: int,
                   k_scale_sigma: Optional[float] = None):
    """q [N, h_q, D], k / v [N, h_kv, D] bf16 bits for a whole sequence [prefix ; branches]
    (N = prefix_len + sum(branch_lens)), seeded N(0, 1) like the decode workloads."""
    rng = np.random.default_rng(seed)
    N = int(prefix_len) + int(np.sum(branch_lens))
    q = _normal(rng, (N, h_q, head_dim))
    k = _normal(rng, (N, h_kv, head_dim))
    v = _normal(rng, (N, h_kv, head_dim))
    if k_scale_sigma is not None:
        k = k * rng.lognormal(0.0, k_scale_sigma, size=(1, h_kv, head_dim)).astype(np.float32)
    return f32_to_bf16_bits(q), f32_to_bf16_bits(k), f32_to_bf16_bits(v)
