"""GPU parity of the fp32 CUDA-core decode (PIC_PREC_FP32) against the fp64
oracle, element by element on the same seeded inputs, through the C ABI.

Bar: max |GPU - oracle| <= 1e-4 on [0, 1] RGB, on every pixel: whole images
for c1-c3, the whole 3840x2160 image for c4, and all 64 images of the c5
batch decoded in one launch (the launch configuration the benchmark times).
"""
import numpy as np
import pytest

from paper_2609_09020_gb300 import workloads as wk

from decode_util import TOL, gpu_decode, max_abs_diff, oracle_full

pytestmark = pytest.mark.gpu
P = "fp32"


@pytest.fixture(scope="module", autouse=True)
def _built():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_09020_gb300 import build
    build.build()


def _check_full(orc, wl, clamp=True, tol=TOL[P]):
    x = wk.make_inputs(wl)
    got = gpu_decode(wl, x, P, clamp=clamp)
    for b in range(x.latents.shape[0]):
        want = oracle_full(orc, wl, x, b, P, clamp=clamp)
        if clamp:
            d, where = max_abs_diff(got[b], want)
            assert d <= tol, (wl.name, b, d, where)
        else:  # raw MLP output: relative to the magnitude
            d, where = max_abs_diff(got[b], want)
            scale = max(1.0, float(np.abs(want).max()))
            assert d <= tol * scale, (wl.name, b, d, where, scale)
    return got


@pytest.mark.parametrize("name", ["c1", "c2", "c3"])
def test_full_image(orc, name):
    _check_full(orc, wk.WORKLOADS[name])


@pytest.mark.parametrize("name", ["c1", "c2"])
def test_full_image_unclamped(orc, name):
    _check_full(orc, wk.WORKLOADS[name], clamp=False)


@pytest.mark.parametrize("name", ["c4", "c5"])
def test_full_size_every_pixel(orc, name):
    """c4 (3840x2160) and c5 (64 images in one launch): every pixel of every
    image, including the 128-pixel tile seams of the 3840-wide rows."""
    got = _check_full(orc, wk.WORKLOADS[name])
    assert got.min() >= 0.0 and got.max() <= 1.0


# Edge and ragged shapes: 1-pixel images, sizes that are not multiples of the
# 128-pixel tile or of 2^l, deep pyramids whose coarse levels are 1 x 1.
EDGE = [
    wk.custom("e1x1", 1, 1, 1, 1, (1, 16, 16, 3)),
    wk.custom("e3x17", 3, 17, 3, 1, (3, 16, 16, 3), act="gelu"),
    wk.custom("e17x33", 17, 33, 5, 2, (10, 40, 40, 3)),
    wk.custom("e33x129", 33, 129, 7, 1, (7, 64, 64, 3)),
    wk.custom("e5x300", 5, 300, 4, 1, (4, 16, 16, 3), clip=63, lap_scale=8.0),
    wk.custom("tall", 257, 3, 8, 2, (16, 64, 64, 64, 3), act="gelu"),
]


@pytest.mark.parametrize("wl", EDGE, ids=lambda w: w.name)
def test_edge_shapes(orc, wl):
    _check_full(orc, wl)


# Ragged shapes on every specialised architecture, with the kernel each one
# must run on: the register-tiled contraction (a hidden layer wider than 16;
# a row's last tile is partly past the image edge) and the one-thread-per-
# pixel kernel (nets no wider than 16).  The batched cases put many images
# into one CTA's tile range, so the weights are reloaded mid-range.
EDGE_SPECIALISED = [
    (wk.custom("c2arch_9x200", 9, 200, 7, 1, (7, 40, 40, 3), act="gelu"), "fp32_7x40x40x3_gelu"),
    (wk.custom("c3arch_7x130", 7, 130, 7, 2, (14, 64, 64, 3)), "fp32_14x64x64x3_relu"),
    (wk.custom("c4arch_5x383", 5, 383, 8, 2, (16, 64, 64, 64, 3), act="gelu", clip=63,
               lap_scale=4.0), "fp32_16x64x64x64x3_gelu"),
    (wk.custom("w32arch_6x250", 6, 250, 8, 1, (8, 32, 32, 32, 3)), "fp32_8x32x32x32x3_relu"),
    (wk.custom("w64arch_3x131", 3, 131, 8, 1, (8, 64, 64, 64, 3)), "fp32_8x64x64x64x3_relu"),
    (wk.custom("w8arch_4x140", 4, 140, 8, 1, (8, 8, 8, 8, 3)), "fp32_8x8x8x8x3_relu"),
    (wk.custom("w16arch_2x77", 2, 77, 8, 1, (8, 16, 16, 16, 3)), "fp32_8x16x16x16x3_relu"),
    (wk.custom("c5arch_x40_2x129", 2, 129, 7, 1, (7, 64, 64, 3), seed=30, batch=40),
     "fp32_7x64x64x3_relu"),
    (wk.custom("c1arch_x24_3x5", 3, 5, 4, 1, (4, 16, 16, 3), seed=70, batch=24), "fp32_4x16x16x3_relu"),
]


@pytest.mark.parametrize("wl,kernel", EDGE_SPECIALISED, ids=lambda c: getattr(c, "name", c))
def test_edge_shapes_specialised(orc, wl, kernel):
    from paper_2609_09020_gb300.pic import Decoder
    dec = Decoder.for_workload(wl, P, max_batch=len(wl.seeds))
    assert dec.kernel_name == kernel
    dec.close()
    _check_full(orc, wl)


def test_generic_kernel_arch(orc):
    """An arch with no compile-time specialisation runs on the generic kernel."""
    from paper_2609_09020_gb300.pic import Decoder
    wl = wk.custom("gen", 19, 45, 3, 2, (6, 24, 12, 3), act="gelu", seed=3)
    dec = Decoder.for_workload(wl, P)
    assert dec.kernel_name == "fp32_generic"
    dec.close()
    _check_full(orc, wl)


def test_batch_images_are_independent(orc):
    wl = wk.WORKLOADS["c2"].replace(seeds=(5, 6, 7), name="c2x3")
    x = wk.make_inputs(wl)
    got = gpu_decode(wl, x, P)
    for b in range(3):
        d, _ = max_abs_diff(got[b], oracle_full(orc, wl, x, b, P))
        assert d <= TOL[P]
    assert not np.array_equal(got[0], got[1])


def test_host_buffer_entry_point_matches_device_path():
    wl = wk.WORKLOADS["c1"].replace(seeds=(0, 1), name="c1x2")
    x = wk.make_inputs(wl)
    a = gpu_decode(wl, x, P)
    b = gpu_decode(wl, x, P, batch_host=True)
    assert np.array_equal(a, b)


def test_specialised_kernels_are_selected():
    from paper_2609_09020_gb300.pic import Decoder
    for name in ("c1", "c2", "c3", "c4", "c5"):
        wl = wk.WORKLOADS[name]
        dec = Decoder.for_workload(wl, P)
        assert dec.kernel_name.startswith("fp32_") and dec.kernel_name != "fp32_generic"
        dec.close()


def test_bad_calls_launch_nothing():
    """Rejected calls return an error and leave the output untouched."""
    import torch
    from paper_2609_09020_gb300 import pic
    from paper_2609_09020_gb300.pic import Decoder
    wl = wk.WORKLOADS["c1"]
    x = wk.make_inputs(wl)
    dec = Decoder.for_workload(wl, P)
    dev = torch.device("cuda:0")
    lat = torch.from_numpy(x.latents).to(dev)
    st = torch.from_numpy(x.steps).to(dev)
    w = torch.from_numpy(x.weights_for(P)).to(dev)
    out = torch.full((1, 3, wl.H, wl.W), -7.0, device=dev)
    s = torch.cuda.current_stream().cuda_stream
    h = dec.handle
    assert pic.pic_decode(h, lat.data_ptr(), st.data_ptr(), w.data_ptr(), wl.H + 1, wl.W,
                          out.data_ptr(), s) == pic.PIC_ERR_INVALID_ARG
    assert pic.pic_decode(h, lat.data_ptr(), st.data_ptr(), w.data_ptr(), wl.H, 0,
                          out.data_ptr(), s) == pic.PIC_ERR_INVALID_ARG
    assert pic.pic_decode(h, lat.data_ptr() + 4, st.data_ptr(), w.data_ptr(), wl.H, wl.W,
                          out.data_ptr(), s) == pic.PIC_ERR_INVALID_ARG
    assert pic.pic_decode_batch(h, 2, lat.data_ptr(), st.data_ptr(), w.data_ptr(), wl.H, wl.W,
                                out.data_ptr(), s) == pic.PIC_ERR_INVALID_ARG
    assert pic.pic_decode(h, None, st.data_ptr(), w.data_ptr(), wl.H, wl.W, out.data_ptr(),
                          s) == pic.PIC_ERR_INVALID_ARG
    torch.cuda.synchronize()
    assert bool((out == -7.0).all())
    # a good call on a buffer with a canary tail writes exactly 3 H W floats
    big = torch.full((3 * wl.H * wl.W + 64,), -7.0, device=dev)
    assert pic.pic_decode(h, lat.data_ptr(), st.data_ptr(), w.data_ptr(), wl.H, wl.W,
                          big.data_ptr(), s) == pic.PIC_OK
    torch.cuda.synchronize()
    assert bool((big[-64:] == -7.0).all()) and bool((big[:-64] >= 0).all())
    dec.check()
    dec.close()
