"""pic_decode_batch_host runs copy-in, decode and copy-out of chunks of
images on three streams; its output must be bit-identical to the device
path (same kernels), for batch sizes that end inside the first chunks (one
image, then two), that do not divide into the remaining chunks, weight blobs
whose size makes per-chunk offsets unaligned, and every output and latent
format."""
import numpy as np
import pytest

from paper_2609_09020_gb300 import workloads as wk

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_09020_gb300 import build
    build.build()


def _both(wl, precision, output="f32_chw", latent="int32", B=None, max_batch=None):
    import torch
    from paper_2609_09020_gb300.pic import Decoder
    x = wk.make_inputs(wl)
    B = B or x.latents.shape[0]
    lat = np.ascontiguousarray(x.latents[:B])
    if latent == "fp32":
        lat = np.ascontiguousarray(lat.astype(np.float32) * 0.5)
    st = np.ascontiguousarray(x.steps[:B])
    w = np.ascontiguousarray(x.weights_for(precision)[:B])
    dec = Decoder.for_workload(wl, precision, max_batch=max_batch or B, latent=latent, output=output)
    dt = np.uint8 if output == "u8_hwc" else np.float32
    shape = (B, 3, wl.H, wl.W) if output == "f32_chw" else (B, wl.H, wl.W, 3)
    host = torch.from_numpy(np.zeros(shape, dtype=dt)).pin_memory()
    pin = [torch.from_numpy(a).pin_memory() for a in (lat, st, w)]
    dec.decode_batch_host(pin[0], pin[1], pin[2], wl.H, wl.W, host, B=B)
    dev = torch.zeros(shape, dtype=torch.uint8 if dt == np.uint8 else torch.float32, device="cuda")
    dec.decode_batch(pin[0].cuda(), pin[1].cuda(), pin[2].cuda(), wl.H, wl.W, dev, B=B)
    dec.check()
    dec.close()
    return host.numpy(), dev.cpu().numpy()


@pytest.mark.parametrize("B", [1, 2, 3, 5, 13, 17, 64])
def test_host_pipeline_equals_device_path_tc(B):
    got, ref = _both(wk.WORKLOADS["c5"], "fp16_tc", B=B, max_batch=64)
    assert np.array_equal(got, ref)


def test_host_pipeline_unaligned_blobs_fp32():
    # 5-7-7-3: 101 weights per image and 3 x 33 x 51 outputs (odd sizes)
    wl = wk.custom("h", H=33, W=51, L=5, C=1, dims=(5, 7, 7, 3), act="gelu", batch=11)
    got, ref = _both(wl, "fp32")
    assert np.array_equal(got, ref)


@pytest.mark.parametrize("output", ["u8_hwc", "f32_hwc"])
def test_host_pipeline_outputs_and_fp32_latents(output):
    wl = wk.custom("h2", H=67, W=130, L=4, C=1, dims=(4, 16, 16, 3), batch=9)
    got, ref = _both(wl, "fp16_tc", output=output, latent="fp32")
    assert np.array_equal(got, ref)
