"""Host-side buffer checks of the Python Decoder (no GPU): the C ABI gets bare
pointers, so the wrapper refuses undersized, non-contiguous or misplaced
buffers before anything launches.  Sizes are counted here by hand."""
import numpy as np
import pytest
import torch


@pytest.fixture(scope="module")
def pic():
    from paper_2609_09020_gb300 import build, pic
    build.build()
    pic.load_library()
    return pic


class _FakeCuda:
    """Stands in for a CUDA tensor: only the metadata the checks read."""

    def __init__(self, nbytes, contiguous=True, index=0):
        self._n, self._c, self.is_cuda = nbytes, contiguous, True
        self.device = torch.device("cuda", index)

    def numel(self):
        return self._n

    def element_size(self):
        return 1

    def is_contiguous(self):
        return self._c


def test_bytes_of_the_768x512_batch(pic):
    # 7 single-channel levels of 768x512: 768x512 + 384x256 + ... + 12x8
    n_lat = sum((768 >> l) * (512 >> l) for l in range(7))
    assert n_lat == 524256
    arch = pic.make_arch(7, 1, (7, 64, 64, 3), "relu", "fp16_tc", True, 512, 768, 64)
    need = pic.decode_buffer_bytes(arch, 64, 512, 768)
    n_par = 64 * 8 + 64 * 65 + 3 * 65
    assert need == {"latents": 4 * 64 * n_lat, "steps": 4 * 64 * 7,
                    "weights": 2 * 64 * n_par, "out": 4 * 3 * 64 * 512 * 768}


def test_bytes_follow_the_formats(pic):
    # ceil-sized levels (1080 -> 540, 270, 135), two channels, fp32 weights,
    # fp32 latents (no steps), uint8 output
    arch = pic.make_arch(4, 2, (8, 16, 3), "gelu", "fp32", True, 1080, 1920, 2,
                         latent="fp32", output="u8_hwc")
    need = pic.decode_buffer_bytes(arch, 2, 1080, 1920)
    n_lat = 2 * (1920 * 1080 + 960 * 540 + 480 * 270 + 240 * 135)
    assert need == {"latents": 4 * 2 * n_lat, "steps": 0,
                    "weights": 4 * 2 * (16 * 9 + 3 * 17), "out": 3 * 2 * 1080 * 1920}
    arch.output_format = pic.PIC_OUT_F32_HWC
    assert pic.decode_buffer_bytes(arch, 2, 1080, 1920)["out"] == 4 * 3 * 2 * 1080 * 1920


def test_checks_refuse_bad_buffers(pic):
    need = {"latents": 64, "steps": 16, "weights": 32, "out": 48}
    ok = {k: _FakeCuda(v) for k, v in need.items()}
    pic.check_decode_buffers(need, 1, 2, 2, **ok)
    for name in need:
        with pytest.raises(ValueError, match=name):
            pic.check_decode_buffers(need, 1, 2, 2, **{**ok, name: _FakeCuda(need[name] - 1)})
        with pytest.raises(ValueError, match="contiguous"):
            pic.check_decode_buffers(need, 1, 2, 2,
                                     **{**ok, name: _FakeCuda(need[name], contiguous=False)})
        with pytest.raises(ValueError, match="CUDA"):  # a host tensor on the device path
            pic.check_decode_buffers(need, 1, 2, 2,
                                     **{**ok, name: torch.zeros(need[name], dtype=torch.uint8)})
        with pytest.raises(ValueError, match="required"):
            pic.check_decode_buffers(need, 1, 2, 2, **{**ok, name: None})
    # steps may be absent where the decoder reads none (fp32 latents)
    pic.check_decode_buffers({**need, "steps": 0}, 1, 2, 2, **{**ok, "steps": None})


def test_host_path_takes_host_buffers(pic):
    need = {"latents": 64, "steps": 16, "weights": 32, "out": 48}
    host = {k: np.zeros(v, np.uint8) for k, v in need.items()}
    pic.check_decode_buffers(need, 1, 2, 2, host=True, **host)
    pic.check_decode_buffers(need, 1, 2, 2, host=True,
                             **{**host, "out": torch.zeros(12, dtype=torch.float32)})
    with pytest.raises(ValueError, match="host"):
        pic.check_decode_buffers(need, 1, 2, 2, host=True, **{**host, "out": _FakeCuda(48)})
    with pytest.raises(ValueError, match="contiguous"):
        pic.check_decode_buffers(need, 1, 2, 2, host=True,
                                 **{**host, "latents": np.zeros((8, 16), np.uint8)[:, ::2]})
    with pytest.raises(ValueError, match="weights"):
        pic.check_decode_buffers(need, 1, 2, 2, host=True,
                                 **{**host, "weights": np.zeros(7, np.float32)})


def test_device_buffers_must_be_on_the_decoders_gpu(pic):
    """A tensor on another GPU than the handle's would be launched on with the
    handle's setup: the wrapper refuses it (the C ABI refuses a call made
    while another device is current)."""
    need = {"latents": 64, "steps": 16, "weights": 32, "out": 48}
    ok = {k: _FakeCuda(v, index=1) for k, v in need.items()}
    pic.check_decode_buffers(need, 1, 2, 2, device=1, **ok)
    pic.check_decode_buffers(need, 1, 2, 2, **ok)  # no device given: not checked
    for name in need:
        with pytest.raises(ValueError, match="cuda:0"):
            pic.check_decode_buffers(need, 1, 2, 2, device=1,
                                     **{**ok, name: _FakeCuda(need[name], index=0)})
