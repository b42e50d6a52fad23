"""Whole-sequence forward attention under the event-factorized mask (Sec. 3.4, Fig. 3)
through the C ABI, against the fp64 oracle.  Same bar as the decode path: max-abs <= 1e-2,
relative-L2 <= 2e-3, LSE within 1e-3."""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2607_02963_gb300 import binding as B
from paper_2607_02963_gb300 import synth

pytestmark = pytest.mark.gpu

MAX_ABS, REL_L2, LSE_ABS = 1e-2, 2e-3, 1e-3


@pytest.fixture(scope="module", autouse=True)
def _cuda(padlib):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.init()


def _dev(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).cuda()


def _run(prefix, lens, h_q, h_kv, D, seed, out_dtype=0, heads=None, sigma=None, flags=0):
    qb, kb, vb = synth.prefill_inputs(seed, prefix, lens, h_q, h_kv, D, k_scale_sigma=sigma)
    N = qb.shape[0]
    prob = B.make_problem(h_q, h_kv, D, 16, 1.0 / math.sqrt(D), out_dtype=out_dtype, flags=flags)
    out = torch.empty((N, h_q, D), dtype=torch.float32 if out_dtype == 0 else torch.bfloat16, device="cuda")
    lse = torch.empty((N, h_q), dtype=torch.float32, device="cuda")
    B.pad_prefill_attn(prob, prefix, lens, _dev(qb), _dev(kb), _dev(vb), out, lse)
    torch.cuda.synchronize()
    B.pad_prefill_status()
    ro, rl = oracle.prefill_attention(oracle.bf16_to_f64(qb), oracle.bf16_to_f64(kb), oracle.bf16_to_f64(vb),
                                      prefix, lens, 1.0 / math.sqrt(D), heads=heads)
    go, gl = out.float().cpu().numpy(), lse.cpu().numpy()
    hs = list(range(h_q)) if heads is None else heads
    go, gl, ro, rl = go[:, hs], gl[:, hs], ro[:, hs], rl[:, hs]
    assert np.all(np.isfinite(go))
    err = np.abs(go - ro)
    assert err.max() <= MAX_ABS, err.max()
    assert np.linalg.norm(go - ro) / np.linalg.norm(ro) <= REL_L2 + (2.0 ** -9 if out_dtype else 0)
    assert np.abs(gl - rl).max() <= LSE_ABS


@pytest.mark.parametrize("prefix,lens", [
    (300, [5, 0, 70, 1, 129]),      # ragged branches, one empty, tiles straddling branches
    (257, []),                      # no branches: plain causal attention
    (0, [40, 90]),                  # no shared prefix
    (64, [64, 64]),                 # every boundary on a tile edge
    (1000, [42] * 13),              # the paper's average: 13 events of ~42 caption tokens
])
@pytest.mark.parametrize("flags", [0, B.FLAG_PREFIX_MMA])
def test_prefill_matches_oracle_d128(prefix, lens, flags):
    """head_dim 128 on the tensor-core kernel (default) and on the warp-level kernel."""
    _run(prefix, lens, 28, 4, 128, seed=prefix + len(lens), flags=flags)


def test_prefill_d64_and_bf16_output():
    _run(200, [3, 17, 66], 8, 2, 64, seed=5)
    _run(200, [3, 17, 66], 8, 2, 64, seed=6, out_dtype=1)


def test_prefill_long_prefix_sampled_heads():
    """An 8k-token prefix with 13 branches (outlier K channels); two heads checked."""
    _run(8192, [42] * 13, 28, 4, 128, seed=7, heads=[0, 27], sigma=0.5)


def test_prefill_tc_group_sizes_and_bf16():
    """Other GQA groups on the tensor-core kernel (128 / G tokens per CTA), bf16 output."""
    _run(500, [30, 2, 77], 8, 2, 128, seed=8)            # G = 4: 32 tokens per CTA
    _run(500, [30, 2, 77], 16, 1, 128, seed=9)           # G = 16: 8 tokens per CTA
    _run(500, [30, 2, 77], 28, 4, 128, seed=10, out_dtype=1)
