"""GPU parity at the largest image sides the C ABI accepts (65536): a
65536-pixel-wide strip (512 tiles per row) and a 65536-pixel-tall column
three pixels wide, on the 64-image workload's net (7-64-64-3: the
register-tiled fp32 kernel and the tensor-core kernel) and on c1's
(4-16-16-3: the one-thread-per-pixel fp32 kernel and its tensor-core
kernel), every pixel against the oracle."""
import numpy as np
import pytest

from paper_2609_09020_gb300 import workloads as wk

from decode_util import TOL, gpu_decode, max_abs_diff, oracle_full

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_09020_gb300 import build
    build.build()


SHAPES = [
    wk.custom("wide_65536", 2, 65536, 7, 1, (7, 64, 64, 3), weight_dtype="fp16", seed=41,
              precisions=("fp32", "fp16_tc")),
    wk.custom("tall_65536", 65536, 3, 7, 1, (7, 64, 64, 3), weight_dtype="fp16", seed=42,
              precisions=("fp32", "fp16_tc")),
    wk.custom("wide_65536_c1net", 1, 65536, 4, 1, (4, 16, 16, 3), seed=43,
              precisions=("fp32", "fp16_tc")),
]


@pytest.mark.parametrize("precision", ["fp32", "fp16_tc"])
@pytest.mark.parametrize("wl", SHAPES, ids=lambda w: w.name)
def test_largest_sides(orc, wl, precision):
    x = wk.make_inputs(wl)
    got = gpu_decode(wl, x, precision)
    want = oracle_full(orc, wl, x, 0, precision)
    d, where = max_abs_diff(got[0], want)
    assert d <= TOL[precision], (wl.name, precision, d, where)
