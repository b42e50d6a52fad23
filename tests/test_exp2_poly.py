"""Error bound of the FMA-pipe 2^x used for part of the softmax exponentials in the
tensor-core prefix kernels: the constants are read from the kernels' shared header and the
instruction sequence (Cody-Waite split, cubic, exponent insertion) is replayed in fp32."""
import os
import re

import numpy as np

SRC = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))),
                   "paper_2607_02963_gb300", "csrc", "pad_tc_common.cuh")


def constants():
    txt = open(SRC).read()
    return [np.float32(float(re.search(rf"kExpC{i} = ([0-9.eE+-]+)f;", txt).group(1))) for i in range(4)]


def emulate(x):
    c0, c1, c2, c3 = constants()
    x = np.maximum(x.astype(np.float32), np.float32(-125.0))
    magic = np.float32(12582912.0)
    t = (magic + np.floor(x)).astype(np.float32)       # add.rm: exact for |x| < 2^22
    n = (t - magic).astype(np.float32)
    f = (x - n).astype(np.float32)
    q = (f * c3 + c2).astype(np.float32)
    q = (f * q + c1).astype(np.float32)
    q = (f * q + c0).astype(np.float32)
    bits = q.view(np.uint32) + (t.view(np.uint32) << np.uint32(23))
    return bits.view(np.float32)


def test_relative_error_below_bf16_rounding():
    x = np.linspace(-125.0, 8.0, 3_000_001, dtype=np.float32)
    rel = emulate(x).astype(np.float64) / np.exp2(x.astype(np.float64)) - 1.0
    assert np.abs(rel).max() < 2.5e-4          # bf16 rounding of P is up to 2^-9 = 2e-3


def test_exact_at_integers_and_monotone():
    x = np.arange(-125, 9, dtype=np.float32)
    y = emulate(x).astype(np.float64)
    np.testing.assert_allclose(y, np.exp2(x.astype(np.float64)), rtol=1e-4)
    xs = np.linspace(-20, 8, 200001, dtype=np.float32)
    assert np.all(np.diff(emulate(xs)) >= 0)


def test_clamp_keeps_tiny_results_normal():
    y = emulate(np.array([-500.0, -127.5, -125.0], dtype=np.float32))
    assert np.all(y >= 2.0 ** -126) and np.all(y < 2.0 ** -124)
