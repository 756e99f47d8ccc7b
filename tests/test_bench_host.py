"""The bench's roofline arithmetic on the host: algorithmic work per launch
from first principles (unpadded MACs; int32 latents, weights, steps and fp32
RGB bytes moved once), and the binding time of the 64-image workload."""
import importlib.util
import os

import pytest

from paper_2609_09020_gb300 import workloads as wk

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def bench():
    spec = importlib.util.spec_from_file_location("bench_mod", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def _level(n, l):
    return -(-n // (1 << l))


def test_c5_algorithmic_work(bench):
    wl = wk.WORKLOADS["c5"]
    B = 64
    flops, nbytes = bench.algorithmic(wl, B)
    px = B * 768 * 512
    macs = 7 * 64 + 64 * 64 + 64 * 3  # 7-64-64-3, biases excluded
    assert macs == 4736
    assert flops == 2 * macs * px == 238_370_684_928
    latents = sum(_level(512, l) * _level(768, l) for l in range(7)) * 4   # int32, one channel
    weights = (7 * 64 + 64 + 64 * 64 + 64 + 64 * 3 + 3) * 2               # fp16, with biases
    steps = 7 * 4
    rgb = 3 * 768 * 512 * 4
    assert B * latents == 134_209_536 and B * weights == 622_976 and B * rgb == 301_989_888
    assert nbytes == B * (latents + weights + steps + rgb)


def test_c5_binding_time(bench):
    """max(FLOPs / 1892.3 TFLOP/s, bytes / 6787.6 GB/s) = 126.0 us (tensor-bound)."""
    flops, nbytes = bench.algorithmic(wk.WORKLOADS["c5"], 64)
    t_tc, t_hbm = flops / 1892.3e12, nbytes / 6787.6e9
    assert t_tc > t_hbm
    assert abs(t_tc * 1e6 - 125.97) < 0.05
    assert abs(t_hbm * 1e6 - 64.36) < 0.05


def test_whole_job_rate_counts_every_rank(bench):
    # weak scaling: 2 ranks x 64 images of 768x512 in 1 ms -> 2 x 25.17 M px / 1 ms
    assert abs(bench.whole_job_rate(64 * 768 * 512, 2, 1.0) - 2 * 64 * 768 * 512 / 1e3) < 1e-6


def test_executed_tensor_work_per_pixel(bench):
    """MACs the tensor path executes, counted by hand from the kernel's
    operand layout (hi and lo halves of K, one K = 16 bias step per hidden
    and output layer, N padded to 16)."""
    # c5 7-64-64-3: layer 0 K = 16 (7 hi + 7 lo + bias, padded) x N 64; hidden
    # K = 64 + 64 + 16; output layer on the tensor cores, N = 16
    assert bench.executed_tensor_macs_per_px(wk.WORKLOADS["c5"]) == 16 * 64 + 144 * 64 + 144 * 16 == 12544
    # c4 16-64-64-64-3: layer 0 K = 48 (33 padded); two hidden layers; output on the CUDA cores
    assert bench.executed_tensor_macs_per_px(wk.WORKLOADS["c4"]) == 48 * 64 + 2 * 144 * 64
    # c2 7-40-40-3: N padded to 48, so the output layer stays on the tensor cores
    assert bench.executed_tensor_macs_per_px(wk.WORKLOADS["c2"]) == 16 * 48 + 112 * 48 + 112 * 16
    assert not bench.tc_output_on_tensor_cores(wk.WORKLOADS["c1"])  # width 16: CUDA cores
    assert bench.tc_output_on_tensor_cores(wk.WORKLOADS["c3"])


def test_activation_inclusive_alu_work_per_pixel(bench):
    """FP32-pipe operations per pixel behind the activation-inclusive bound."""
    g = bench.GELU_FP32_OPS
    assert g == 13  # z^2, 5 + 4 Horner steps, P * (1 / Q), the saturating fma, z * Phi
    # c4 on the tensor path: 192 GELUs, the split of the two hidden layers
    # feeding MMAs (2 per value), the 64 x 3 output layer on the CUDA cores
    assert bench.alu_ops_per_px(wk.WORKLOADS["c4"], "fp16_tc") == 192 * g + 2 * 128 + 3 * 64 == 2944
    # c5 (ReLU) on the tensor path: the split of both hidden layers only
    assert bench.alu_ops_per_px(wk.WORKLOADS["c5"], "fp16_tc") == 2 * 128
    # c2 on the fp32 path: 80 GELUs plus every MLP MAC (7*40 + 40*40 + 40*3)
    assert bench.alu_ops_per_px(wk.WORKLOADS["c2"], "fp32") == 80 * g + 2000
