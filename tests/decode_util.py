"""Helpers shared by the GPU parity tests: run the CUDA path through the C ABI
binding, run the fp64 oracle on the same inputs, compare."""
from __future__ import annotations

import os

import numpy as np

from paper_2609_09020_gb300 import workloads as wk

# Tolerances on [0, 1] RGB, max |GPU - oracle| (the decode's stated bars).
TOL = {"fp32": 1e-4, "fp16_tc": 4e-3, "fp16_tc_lo8": 4e-3}
# Oracle threads: the host cores of whatever machine runs the tests.
ORACLE_THREADS = max(1, min(16, os.cpu_count() or 1))


def gpu_decode(wl: wk.Workload, x: wk.Inputs, precision: str, clamp: bool = True,
               batch_host: bool = False, staging: str = "auto") -> np.ndarray:
    """Decodes every image of x on the GPU; returns fp32 [B][3][H][W] (host)."""
    import torch
    from paper_2609_09020_gb300.pic import Decoder
    dec = Decoder.for_workload(wl, precision, clamp=clamp, max_batch=x.latents.shape[0],
                               staging=staging)
    B = x.latents.shape[0]
    w = x.weights_for(precision)
    if batch_host:
        out = np.empty((B, 3, wl.H, wl.W), dtype=np.float32)
        dec.decode_batch_host(np.ascontiguousarray(x.latents), np.ascontiguousarray(x.steps),
                              np.ascontiguousarray(w), wl.H, wl.W, out)
        dec.check()
        dec.close()
        return out
    dev = torch.device("cuda:0")
    lat = torch.from_numpy(np.ascontiguousarray(x.latents)).to(dev)
    steps = torch.from_numpy(np.ascontiguousarray(x.steps)).to(dev)
    wt = torch.from_numpy(np.ascontiguousarray(w)).to(dev)
    out = torch.full((B, 3, wl.H, wl.W), float("nan"), dtype=torch.float32, device=dev)
    dec.decode_batch(lat, steps, wt, wl.H, wl.W, out, B=B)
    dec.check()
    torch.cuda.synchronize()
    res = out.cpu().numpy()
    dec.close()
    return res


def oracle_full(orc, wl: wk.Workload, x: wk.Inputs, b: int, precision: str,
                clamp: bool = True, defined: bool = False) -> np.ndarray:
    """The oracle's decode of image b with the weights the GPU path consumes
    (``x.weights_for(precision)``), or, with defined=True, with the weights
    the workload defines (its fp32 draw where the tensor path gets an fp16
    copy of it)."""
    w = x.oracle_weights(precision) if defined else x.weights_for(precision)
    return orc.decode(x.latents[b], x.steps[b].astype(np.float64),
                      w[b].astype(np.float64), wl.H, wl.W, wl.L, wl.C,
                      wl.dims, wl.act, clamp=clamp, nthreads=ORACLE_THREADS)


def oracle_pixels(orc, wl, x, b, precision, pix, clamp=True) -> np.ndarray:
    """Oracle values [n][3] at flat pixel indices pix of image b."""
    return orc.decode_pixels(x.latents[b], x.steps[b].astype(np.float64),
                             x.weights_for(precision)[b].astype(np.float64), wl.H, wl.W, wl.L,
                             wl.C, wl.dims, wl.act, pix, clamp=clamp)


def max_abs_diff(got: np.ndarray, want: np.ndarray):
    d = np.abs(got.astype(np.float64) - want)
    d = np.where(np.isnan(d), np.inf, d)
    i = int(np.argmax(d))
    return float(d.ravel()[i]), np.unravel_index(i, d.shape)


def psnr(a: np.ndarray, b: np.ndarray) -> float:
    mse = float(np.mean((a.astype(np.float64) - b) ** 2))
    return float("inf") if mse == 0 else 10 * np.log10(1.0 / mse)
