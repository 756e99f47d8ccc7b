"""The fp64 oracle against its pins (closed forms, brute force, hand-computed
values); see tests/oracle_pins.py."""
import pytest

import oracle_pins


@pytest.mark.parametrize("pin", oracle_pins.PINS, ids=lambda f: f.__name__)
def test_pin(orc, pin):
    pin(orc)


def test_upsample_matches_torch_interpolate(orc):
    """Cross-check against an independent implementation: torch's bilinear
    interpolation (half-pixel centres, align_corners=False) in fp64 on CPU."""
    torch = pytest.importorskip("torch")
    import numpy as np
    rng = np.random.Generator(np.random.PCG64(1))
    for (hl, wl, H, W) in [(3, 5, 5, 9), (17, 30, 135, 240), (1, 1, 4, 4), (2, 3, 3, 5),
                           (12, 8, 768, 512), (34, 60, 1080, 1920)]:
        g = rng.standard_normal((hl, wl)) * 10
        want = torch.nn.functional.interpolate(torch.from_numpy(g)[None, None], size=(H, W),
                                               mode="bilinear", align_corners=False)[0, 0].numpy()
        got = orc.upsample(g, H, W)
        assert np.max(np.abs(got - want)) <= 1e-12


def test_gelu_matches_torch(orc):
    torch = pytest.importorskip("torch")
    import numpy as np
    z = np.linspace(-8, 8, 161)
    want = torch.nn.functional.gelu(torch.from_numpy(z), approximate="none").numpy()
    got = np.array([orc.act(v, "gelu") for v in z])
    assert np.max(np.abs(got - want)) <= 1e-14


def test_oracle_rejects_bad_args(orc):
    import numpy as np
    with pytest.raises(ValueError):
        orc.decode(np.zeros(16, np.int32), [1.0], np.zeros(15), 4, 4, 1, 1, [1, 3, 4], "relu")
    with pytest.raises(ValueError):
        orc.decode(np.zeros(15, np.int32), [1.0], np.zeros(6), 4, 4, 1, 1, [1, 3], "relu")


def test_multithreaded_decode_is_identical(orc):
    """Splitting rows over threads does not change any value."""
    import numpy as np
    from paper_2609_09020_gb300 import workloads as wk
    wl = wk.custom("t", H=37, W=53, L=4, C=2, dims=(8, 16, 16, 3), act="gelu", seed=4)
    x = wk.make_inputs(wl)
    args = (x.latents[0], x.steps[0], x.oracle_weights("fp32"), wl.H, wl.W, wl.L, wl.C,
            wl.dims, wl.act)
    a = orc.decode(*args, nthreads=1)
    b = orc.decode(*args, nthreads=4)
    assert np.array_equal(a, b)
