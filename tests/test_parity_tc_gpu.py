"""GPU parity of the tensor-core decode (PIC_PREC_FP16_TC, tcgen05) against
the fp64 oracle on the same seeded inputs, through the C ABI.

Two references per image:
- the decode as defined: the oracle on the weights the workload defines (its
  fp32 draw for c1-c4, whose tensor path consumes an fp16 copy; the fp16
  weights themselves for c5 and the fp16 edge cases).  Bars: max |GPU -
  oracle| <= 4e-3 on [0, 1] RGB and |PSNR(G, T) - PSNR(O, T)| <= 0.02 dB
  against a noisy target T = clamp(O + N(0, sigma^2)) at ~35 dB (the
  paper's operating range).  The fp16 weight copy alone moves the c4 decode
  by up to ~2.6e-3; this is the check of the decode the workload asks for.
- the kernel's own arithmetic: the oracle on the fp16 weights the kernel
  consumes.  The split (hi + lo) operands carry ~22 significant bits, so the
  error is held to SPLIT_BOUND, far below the bar: plain fp16 operands would
  land near 4e-3 on these workloads, and a broken lo-term would show up here.
"""
import numpy as np
import pytest

from paper_2609_09020_gb300 import workloads as wk

from decode_util import TOL, gpu_decode, max_abs_diff, oracle_full, psnr

pytestmark = pytest.mark.gpu
P = "fp16_tc"
SPLIT_BOUND = 2e-4


@pytest.fixture(scope="module", autouse=True)
def _built():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_09020_gb300 import build
    build.build()


def _noisy_target(ref: np.ndarray, seed: int) -> np.ndarray:
    rng = np.random.Generator(np.random.PCG64(seed))
    sigma = 10 ** (-35 / 20)
    return np.clip(ref + rng.normal(0.0, sigma, ref.shape), 0.0, 1.0)


def _check(orc, wl, images=None, clamp=True):
    x = wk.make_inputs(wl)
    got = gpu_decode(wl, x, P, clamp=clamp)
    # the kernel consumes a rounded copy of the defined weights (fp32 draws)
    copy = not np.array_equal(x.weights_for(P).astype(np.float64), x.oracle_weights(P))
    worst = 0.0
    for b in (range(x.latents.shape[0]) if images is None else images):
        want_in = oracle_full(orc, wl, x, b, P, clamp=clamp)  # the kernel's fp16 weights
        want = oracle_full(orc, wl, x, b, P, clamp=clamp, defined=True) if copy else want_in
        scale = 1.0 if clamp else max(1.0, float(np.abs(want).max()))
        d, where = max_abs_diff(got[b], want)
        assert d <= TOL[P] * scale, (wl.name, b, d, where, "bar against the defined weights")
        if clamp:
            t = _noisy_target(want, 1000 + b)
            assert abs(psnr(got[b], t) - psnr(want, t)) <= 0.02, (wl.name, b)
        d_in, where = max_abs_diff(got[b], want_in)
        assert d_in <= SPLIT_BOUND * scale, (wl.name, b, d_in, where, "split-precision bound")
        worst = max(worst, d)
    return worst


def test_c5_all_64_images(orc):
    """The 64-image throughput workload, every pixel of every image."""
    _check(orc, wk.WORKLOADS["c5"])


def test_c4_full_image(orc):
    """3840x2160, 8 levels x 2 channels, 16-64-64-64-3 GELU: every pixel
    against the oracle on the workload's fp32 weights (the 4e-3 / 0.02 dB
    bars), and against the oracle on the fp16 copy the kernel consumes (the
    split-precision bound)."""
    _check(orc, wk.WORKLOADS["c4"])


@pytest.mark.parametrize("name", ["c1", "c2", "c3"])
def test_fp32_workloads_on_tensor_path(orc, name):
    """The other workloads' architectures on the tensor path, with the fp16
    copy of their fp32 weights (widths 16, 40 -> padded 48, and 64 with two
    channels per level)."""
    _check(orc, wk.WORKLOADS[name])


def test_c5_unclamped(orc):
    wl = wk.WORKLOADS["c5"].replace(seeds=(100, 101), name="c5x2")
    _check(orc, wl, clamp=False)


EDGE = [
    wk.custom("t1x1", 1, 1, 7, 1, (7, 64, 64, 3), weight_dtype="fp16", precisions=(P,)),
    wk.custom("t3x200", 3, 200, 7, 1, (7, 64, 64, 3), weight_dtype="fp16", precisions=(P,)),
    wk.custom("t129x131", 129, 131, 7, 1, (7, 64, 64, 3), weight_dtype="fp16", batch=3,
              precisions=(P,)),
    wk.custom("t70x383", 70, 383, 8, 2, (16, 64, 64, 64, 3), act="gelu", clip=63, lap_scale=4.0,
              precisions=(P,)),
]


@pytest.mark.parametrize("wl", EDGE, ids=lambda w: w.name)
def test_edge_shapes(orc, wl):
    _check(orc, wl)


def test_tc_kernels_are_selected():
    from paper_2609_09020_gb300.pic import Decoder
    for name in ("c1", "c2", "c3", "c4", "c5"):
        dec = Decoder.for_workload(wk.WORKLOADS[name], P)
        assert dec.kernel_name.startswith("tc05_")
        dec.close()


def test_repeated_calls_are_deterministic():
    wl = wk.WORKLOADS["c5"].replace(seeds=(100, 101, 102), name="c5x3")
    x = wk.make_inputs(wl)
    a = gpu_decode(wl, x, P)
    b = gpu_decode(wl, x, P)
    assert np.array_equal(a, b)


# Latent staging: the TMA-staged kernels (the tile's full-resolution row as
# TMA boxes) and the per-thread-copy kernels compute the same arithmetic on
# the same words, so their outputs are equal bit for bit; every workload
# architecture runs both, the one PIC_STAGING_AUTO does not pick on top of
# the checks above.
STAGING_CASES = [
    wk.WORKLOADS["c5"].replace(seeds=(100, 101, 102), name="c5x3"),
    wk.WORKLOADS["c4"],
    wk.WORKLOADS["c3"],
    wk.WORKLOADS["c2"],
    wk.WORKLOADS["c1"],
    EDGE[1],  # 3 x 200: one tile per row, ragged tail
    EDGE[2],  # 129 x 131, batch of 3
]


@pytest.mark.parametrize("wl", STAGING_CASES, ids=lambda w: w.name)
def test_tma_and_copy_staging_agree(orc, wl):
    from paper_2609_09020_gb300.pic import Decoder
    x = wk.make_inputs(wl)
    tma = gpu_decode(wl, x, P, staging="tma")
    cp = gpu_decode(wl, x, P, staging="copies")
    assert np.array_equal(tma, cp), wl.name
    want = oracle_full(orc, wl, x, 0, P)  # the kernels' own bound, image 0
    d, where = max_abs_diff(tma[0], want)
    assert d <= SPLIT_BOUND, (wl.name, d, where)
    for staging, suffix in (("tma", "_tma"), ("copies", "")):
        dec = Decoder.for_workload(wl, P, staging=staging)
        assert dec.kernel_name.endswith(suffix) and ("_tma" in dec.kernel_name) == (staging == "tma")
        dec.close()


# The fp8 lo term (PIC_PREC_FP16_TC_LO8, the 7-64-64-3 architecture): the
# hidden operands carry about 15 significant bits (fp16 hi + e4m3 lo, the
# activations scaled by 2^6), so its own bound is wider than the split's.
# A CPU emulation of exactly this arithmetic on 8 of the 64 c5 images
# (tests/test_split_arithmetic.py) reaches 3.4e-4 against the oracle; the
# kernel is held to LO8_BOUND = 1e-3, a quarter of the 4e-3 bar, on top of
# the bar and the PSNR check.
LO8 = "fp16_tc_lo8"
LO8_BOUND = 1e-3


def _check_lo8(orc, wl, clamp=True):
    from paper_2609_09020_gb300.pic import Decoder
    x = wk.make_inputs(wl)
    got = gpu_decode(wl, x, LO8, clamp=clamp)
    dec = Decoder.for_workload(wl, LO8)
    assert dec.kernel_name.endswith("_lo8")
    dec.close()
    worst = 0.0
    for b in range(x.latents.shape[0]):
        want = oracle_full(orc, wl, x, b, P, clamp=clamp)  # fp16 weights: the definition
        scale = 1.0 if clamp else max(1.0, float(np.abs(want).max()))
        d, where = max_abs_diff(got[b], want)
        assert d <= LO8_BOUND * scale, (wl.name, b, d, where)
        if clamp:
            t = _noisy_target(want, 1000 + b)
            assert abs(psnr(got[b], t) - psnr(want, t)) <= 0.02, (wl.name, b)
        worst = max(worst, d)
    return worst


def test_lo8_c5_all_64_images(orc):
    _check_lo8(orc, wk.WORKLOADS["c5"])


def test_lo8_c5_unclamped(orc):
    _check_lo8(orc, wk.WORKLOADS["c5"].replace(seeds=(100, 101), name="c5x2"), clamp=False)


@pytest.mark.parametrize("wl", EDGE[:3], ids=lambda w: w.name)
def test_lo8_edge_shapes(orc, wl):
    _check_lo8(orc, wl)


def test_lo8_needs_its_architecture():
    """Only the 7-64-64-3 ReLU architecture has an fp8-lo kernel."""
    from paper_2609_09020_gb300 import pic
    with pytest.raises(pic.PicError):
        pic.Decoder.for_workload(wk.WORKLOADS["c4"], LO8)
