"""Seeded random shapes through every specialised architecture on both
paths (and random architectures on the generic fp32 kernel), every pixel
against the oracle: image sides from 1 to several tiles with ragged ends,
level counts up to the image's depth, batches whose images share CTA tile
ranges.  The draws are fixed by the seed, so a failure reproduces."""
import numpy as np
import pytest

from paper_2609_09020_gb300 import workloads as wk

from decode_util import TOL, gpu_decode, max_abs_diff, oracle_full

pytestmark = pytest.mark.gpu
SPLIT_BOUND = 2e-4  # the tensor path's own arithmetic against the oracle on its fp16 weights

# (levels, channels, dims, activation, has a tensor-core kernel)
ARCHS = [
    (4, 1, (4, 16, 16, 3), "relu", True),
    (7, 1, (7, 40, 40, 3), "gelu", True),
    (7, 2, (14, 64, 64, 3), "relu", True),
    (8, 2, (16, 64, 64, 64, 3), "gelu", True),
    (7, 1, (7, 64, 64, 3), "relu", True),
    (8, 1, (8, 8, 8, 8, 3), "relu", True),
    (8, 1, (8, 16, 16, 16, 3), "relu", True),
    (8, 1, (8, 32, 32, 32, 3), "relu", True),
    (8, 1, (8, 64, 64, 64, 3), "relu", True),
]


def _cases(n=18, seed=2609):
    rng = np.random.Generator(np.random.PCG64(seed))
    out = []
    for i in range(n):
        if i % 6 == 5:  # a random architecture: the generic fp32 kernel
            L, C = int(rng.integers(1, 6)), int(rng.integers(1, 3))
            hidden = [int(rng.integers(3, 40)) for _ in range(int(rng.integers(1, 4)))]
            arch = (L, C, tuple([L * C] + hidden + [3]), str(rng.choice(["relu", "gelu"])), False)
        else:
            arch = ARCHS[int(rng.integers(len(ARCHS)))]
        L, C, dims, act, tc = arch
        H = int(rng.integers(1, 96))
        W = int(rng.integers(1, 700))
        batch = int(rng.integers(1, 4))
        wl = wk.custom(f"rand{i}_{H}x{W}_b{batch}", H, W, L, C, dims, act=act, weight_dtype="fp16",
                       seed=5000 + 10 * i, batch=batch, precisions=("fp32", "fp16_tc"))
        out.append((wl, "fp32"))
        if tc:
            out.append((wl, "fp16_tc"))
    return out


@pytest.fixture(scope="module", autouse=True)
def _built():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_09020_gb300 import build
    build.build()


@pytest.mark.parametrize("wl,precision", _cases(), ids=lambda c: getattr(c, "name", c))
def test_random_shape(orc, wl, precision):
    x = wk.make_inputs(wl)
    got = gpu_decode(wl, x, precision)
    bound = TOL[precision] if precision == "fp32" else SPLIT_BOUND
    for b in range(x.latents.shape[0]):
        d, where = max_abs_diff(got[b], oracle_full(orc, wl, x, b, precision))
        assert d <= bound, (wl.name, precision, b, d, where)
