"""The rational GELU used by the CUDA path (host-side checks): the committed
header is what the generator produces, the denominator stays >= 1 on the
fitted range (a well-conditioned reciprocal), and the fp32 emulation of the
kernels' evaluation stays within 2e-6 of z Phi(z) everywhere, with the exact
values at the special points: 0 at 0, z beyond the fitted range, 0 far
below it."""
import os

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_header_is_generated_output():
    pytest.importorskip("scipy")
    from paper_2609_09020_gb300 import gen_gelu as g
    with open(os.path.join(ROOT, "paper_2609_09020_gb300", "csrc", "pic_gelu.cuh")) as f:
        committed = f.read()
    assert committed.strip() == g.header(g.fit()).strip()


def test_denominator_is_at_least_one():
    pytest.importorskip("scipy")
    from paper_2609_09020_gb300 import gen_gelu as g
    assert g.min_denominator(g.fit()) >= 1.0


def test_fp32_error_bound():
    pytest.importorskip("scipy")
    from scipy.special import erf
    from paper_2609_09020_gb300 import gen_gelu as g
    pq = g.fit()
    z = np.concatenate([np.linspace(-30, 30, 400001), [0.0, -0.0, 1e-30, -1e-30, 5.5, 5.52]])
    ref = 0.5 * z * (1 + erf(z / np.sqrt(2)))
    got = g.gelu_fp32(z, pq).astype(np.float64)
    assert np.max(np.abs(got - ref)) <= 2e-6
    assert got[np.argmin(np.abs(z))] == 0.0
    # beyond the fitted range Phi saturates: exactly z above, exactly 0 below
    big = np.array([6.0, 9.5, 30.0, 1e4], dtype=np.float32)
    assert np.array_equal(g.gelu_fp32(big, pq), big)
    assert np.all(g.gelu_fp32(-big, pq) == 0.0)
