"""The polynomial GELU used by the CUDA path (host-side checks): the
committed header is what the generator produces, and the fp32 emulation of
its evaluation stays within 2e-6 of z Phi(z) everywhere."""
import os

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_header_is_generated_output():
    pytest.importorskip("scipy")
    from paper_2609_09020_gb300 import gen_gelu_poly as g
    with open(os.path.join(ROOT, "paper_2609_09020_gb300", "csrc", "pic_gelu.cuh")) as f:
        committed = f.read()
    assert committed.strip() == g.header(g.fit()).strip()


def test_fp32_error_bound():
    pytest.importorskip("scipy")
    from scipy.special import erf
    from paper_2609_09020_gb300 import gen_gelu_poly as g
    m = g.fit()
    z = np.concatenate([np.linspace(-30, 30, 400001), [0.0, -0.0, 1e-30, -1e-30, 5.5, 5.52]])
    ref = 0.5 * z * (1 + erf(z / np.sqrt(2)))
    got = g.gelu_fp32(z, m).astype(np.float64)
    assert np.max(np.abs(got - ref)) <= 2e-6
    assert got[np.argmin(np.abs(z))] == 0.0
