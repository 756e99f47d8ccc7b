"""The FP32 FMA microbenchmark (include/pic_measure.h) that the fp32 decode
path's roofline fraction is reported against: a plausible fraction of the
CUDA cores' nominal rate (SMs x 128 lanes x 2 FLOP x clock)."""
import pytest

pytestmark = pytest.mark.gpu


def test_fma_peak_is_plausible():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_09020_gb300 import build, pic
    build.build()
    tf = pic.fma_peak_tflops()
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    nominal = sms * 128 * 2 * 2.2e9 / 1e12  # above any boost clock of the part
    assert 0.3 * nominal < tf < nominal, (tf, nominal)
