"""Grounding readout (Sec. 3.3) through the C ABI against the fp64 oracle.

Bar: segment sums and scores within a relative error derived from fp32 accumulation of
bf16 inputs (|err| <= 1e-4 * sum of magnitudes); the salient set and the interval are
decisions taken from those scores, so they must equal the oracle's wherever the oracle's
score is clear of the threshold by more than that error bound (elsewhere either side is
correct), and every interval must span exactly the kernel's own salient segments; the
aggregated embeddings within 1e-4 relative to their magnitude (fp32 weighted sums).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_02963_gb300 import binding as B
from paper_2607_02963_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda(padlib):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.init()


def _dev_bf16(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).cuda()


def _run(gi, frac):
    T, dp = gi.f_proj.shape
    S = len(gi.offsets) - 1
    K = gi.g_proj.shape[0]
    f, g = _dev_bf16(gi.f_proj), _dev_bf16(gi.g_proj)
    x, emb = _dev_bf16(gi.x), _dev_bf16(gi.g_emb)
    attn = torch.from_numpy(gi.attn).cuda()
    seg = torch.empty((S, dp), dtype=torch.float32, device="cuda")
    scores = torch.empty((K, S), dtype=torch.float32, device="cuda")
    sal = torch.empty((K, S), dtype=torch.uint8, device="cuda")
    iv = torch.empty((K, 2), dtype=torch.int32, device="cuda")
    out = torch.empty((K, gi.x.shape[1]), dtype=torch.float32, device="cuda")
    ws = B.aggregate_workspace(T, S, gi.x.shape[1])
    B.pad_ground_pool(f, gi.offsets, seg)
    B.pad_ground_score(g, seg, frac, scores, sal, iv)
    B.pad_attn_aggregate(x, attn, gi.offsets, iv, emb, out, ws)
    torch.cuda.synchronize()
    # every pooled element is written once and summed in a fixed order: a second call
    # reproduces the output bit for bit
    out2 = torch.empty_like(out)
    B.pad_attn_aggregate(x, attn, gi.offsets, iv, emb, out2, ws)
    torch.cuda.synchronize()
    assert torch.equal(out, out2)
    return seg.cpu().numpy(), scores.cpu().numpy(), sal.cpu().numpy().astype(bool), iv.cpu().numpy(), out.cpu().numpy()


def _check(gi, frac):
    seg, sc, sal, iv, out = _run(gi, frac)
    f64 = oracle.bf16_to_f64(gi.f_proj)
    g64 = oracle.bf16_to_f64(gi.g_proj)
    S = len(gi.offsets) - 1
    # segment sums
    ref_seg = np.stack([f64[gi.offsets[s]:gi.offsets[s + 1]].sum(axis=0) for s in range(S)])
    mag_seg = np.stack([np.abs(f64[gi.offsets[s]:gi.offsets[s + 1]]).sum(axis=0) for s in range(S)])
    assert np.all(np.abs(seg - ref_seg) <= 1e-4 * mag_seg + 1e-6)
    # scores
    ref = oracle.ground_segment_scores(g64, f64, gi.offsets)
    bound = 1e-4 * (np.abs(g64) @ mag_seg.T) + 1e-5
    assert np.all(np.abs(sc - ref) <= bound)
    # decisions, where they are clear
    rsal, riv = oracle.ground_salient(ref, frac)
    best = ref.max(axis=1, keepdims=True)
    ib = bound.max(axis=1, keepdims=True)
    clear = np.abs(ref - frac * best) > 2 * ib * (1 + frac)
    assert np.array_equal(sal[clear], rsal[clear])
    for i in range(sal.shape[0]):
        idx = np.nonzero(sal[i])[0]
        assert idx.size > 0 and iv[i].tolist() == [idx[0], idx[-1]]
        if clear[i].all():
            assert iv[i].tolist() == riv[i].tolist()
    # aggregation, on the kernel's own intervals
    ref_out = oracle.attention_aggregate(oracle.bf16_to_f64(gi.g_emb), oracle.bf16_to_f64(gi.x), gi.attn, iv,
                                         gi.offsets)
    assert np.all(np.abs(out - ref_out) <= 1e-4 * (np.abs(ref_out) + 1.0))
    return sal, iv


@pytest.mark.parametrize("frac", [0.5, 0.7])
@pytest.mark.parametrize("dims", [(3000, 37, 5, 64, 256, 40), (777, 1, 3, 8, 64, 0), (5000, 200, 9, 256, 512, 100)])
def test_grounding_small(dims, frac):
    T, S, K, dp, dm, text = dims
    _check(synth.grounding_inputs(T + S + K, T, S, K, dp, dm, text_tokens=text), frac)


def test_grounding_full_size_long_video():
    """The long_32k video: 32768 prefix tokens (32 text tokens, then 128 two-second
    audio-visual segments), 32 events, projection width 256, hidden size 2048."""
    gi = synth.grounding_inputs(3, 32768, 128, 32, 256, 2048, text_tokens=32)
    sal, iv = _check(gi, 0.5)
    # the event tokens were drawn near their true runs: the best segment lies in them
    hit = [gi.true_seg[i, 0] <= iv[i, 0] <= gi.true_seg[i, 1] or gi.true_seg[i, 0] <= iv[i, 1] <= gi.true_seg[i, 1]
           or (iv[i, 0] <= gi.true_seg[i, 0] and iv[i, 1] >= gi.true_seg[i, 1]) for i in range(32)]
    assert all(hit)


def test_grounding_edge_cases():
    # an empty segment, and an event token pointing away from the features of another
    gi = synth.grounding_inputs(5, 600, 6, 3, 16, 64)
    gi.offsets[3] = gi.offsets[2]
    g = oracle.bf16_to_f64(gi.g_proj)
    g[2] = -g[0] * 4
    gi.g_proj[2] = synth.f32_to_bf16_bits(g[2].astype(np.float32))
    _check(gi, 0.5)
    with pytest.raises(B.PadError):
        B.pad_ground_pool(_dev_bf16(gi.f_proj), np.array([0, 700], np.int32),
                          torch.empty((1, 16), dtype=torch.float32, device="cuda"))


def test_aggregate_long_segment_is_split():
    """A segment of 3000 tokens is pooled in 12 pieces of at most 256 tokens, and a hidden
    size that is not a multiple of 256 leaves a partial column slice; a scratch one float
    short of the documented size is refused."""
    gi = synth.grounding_inputs(9, 3400, 3, 4, 32, 520, text_tokens=0)
    gi.offsets[:] = np.array([0, 200, 3200, 3400], np.int32)
    _check(gi, 0.5)
    ws = B.aggregate_workspace(3400, 3, 520)
    assert ws.numel() == (3 + 14) * 521
    with pytest.raises(B.PadError) as ei:
        B.pad_attn_aggregate(_dev_bf16(gi.x), torch.from_numpy(gi.attn).cuda(), gi.offsets,
                             torch.zeros((4, 2), dtype=torch.int32, device="cuda"), _dev_bf16(gi.g_emb),
                             torch.empty((4, 520), dtype=torch.float32, device="cuda"), ws[:-1])
    assert ei.value.status == 4
