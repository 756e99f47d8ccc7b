"""Output variants (interleaved fp32, interleaved uint8) and the width
ablation's architectures (8-w-w-w-3, w = 8..64, Sec. 4.3) on both decode
paths, against the fp64 oracle through the C ABI."""
import numpy as np
import pytest

from paper_2609_09020_gb300 import workloads as wk

from decode_util import ORACLE_THREADS, TOL, max_abs_diff, oracle_full, oracle_pixels, psnr

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_09020_gb300 import build
    build.build()


def _decode(wl, x, precision, output):
    import torch
    from paper_2609_09020_gb300.pic import Decoder
    B = x.latents.shape[0]
    dec = Decoder.for_workload(wl, precision, max_batch=B, output=output)
    dt = torch.uint8 if output == "u8_hwc" else torch.float32
    shape = (B, 3, wl.H, wl.W) if output == "f32_chw" else (B, wl.H, wl.W, 3)
    out = torch.zeros(shape, dtype=dt, device="cuda")
    dec.decode_batch(torch.from_numpy(x.latents).cuda(), torch.from_numpy(x.steps).cuda(),
                     torch.from_numpy(np.ascontiguousarray(x.weights_for(precision))).cuda(),
                     wl.H, wl.W, out, B=B)
    dec.check()
    res = out.cpu().numpy()
    name = dec.kernel_name
    dec.close()
    return res, name


def _u8_ok(got, want, tol):
    """uint8 from fp32 against the fp64 oracle's bytes: equal, except that
    within the path's tolerance of a rounding boundary either neighbour is
    correct."""
    ref = np.array(np.vectorize(lambda v: int(np.rint(255.0 * min(max(v, 0.0), 1.0))))(want))
    s = 255.0 * np.clip(want, 0.0, 1.0)
    near = np.abs(s - np.floor(s) - 0.5) <= 255.0 * tol
    d = np.abs(got.astype(np.int64) - ref)
    return bool(np.all((d == 0) | (near & (d == 1))))


@pytest.mark.parametrize("precision", ["fp32", "fp16_tc"])
@pytest.mark.parametrize("output", ["f32_hwc", "u8_hwc"])
def test_output_variants(orc, precision, output):
    wl = wk.custom("o", H=97, W=300, L=4, C=1, dims=(4, 16, 16, 3), act="relu", batch=2, seed=70)
    x = wk.make_inputs(wl)
    got, _ = _decode(wl, x, precision, output)
    assert got.shape == (2, 97, 300, 3)
    for b in range(2):
        want = oracle_full(orc, wl, x, b, precision).transpose(1, 2, 0)  # [H][W][3]
        if output == "f32_hwc":
            d, where = max_abs_diff(got[b], want)
            assert d <= TOL[precision], (b, d, where)
        else:
            assert _u8_ok(got[b], want, TOL[precision]), b
            assert orc.to_u8(0.25) == 64  # the conversion both sides define


WIDTHS = [8, 16, 32, 64]


@pytest.mark.parametrize("w", WIDTHS)
@pytest.mark.parametrize("precision", ["fp16_tc", "fp32"])
def test_width_ablation_architectures(orc, w, precision):
    """The whole 64-image batch in one launch (the bench's configuration):
    image 0 checked at every pixel, images 31 and 63 at sampled pixels."""
    wl = wk.WORKLOADS[f"w{w}"]
    x = wk.make_inputs(wl)
    got, name = _decode(wl, x, precision, "f32_chw")
    assert name == ("tc05" if precision == "fp16_tc" else "fp32") + f"_8x{w}x{w}x{w}x3_relu"
    want = oracle_full(orc, wl, x, 0, precision)
    d, where = max_abs_diff(got[0], want)
    assert d <= TOL[precision], (d, where)
    if precision == "fp16_tc":
        rng = np.random.Generator(np.random.PCG64(w))
        t = np.clip(want + rng.normal(0, 10 ** (-35 / 20), want.shape), 0, 1)
        assert abs(psnr(got[0], t) - psnr(want, t)) <= 0.02
    pix = wk.sample_pixels(wl.H, wl.W, 400, w)
    for b in (31, 63):
        ref = oracle_pixels(orc, wl, x, b, precision, pix)
        g = got[b].reshape(3, -1)[:, pix].T
        assert np.abs(g - ref).max() <= TOL[precision], b
