"""A small, self-contained decode run for profilers (ncu): builds the library,
decodes `--images` images of a workload `--launches` times on one stream and
exits.  Inputs are the seeded synthetic workload inputs.

    python -m paper_2609_09020_gb300.profile_case --workload c5 --images 24 --launches 2
"""
from __future__ import annotations

import argparse

import numpy as np


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--workload", default="c5")
    ap.add_argument("--images", type=int, default=0, help="0 = all images of the workload")
    ap.add_argument("--precision", default=None)
    ap.add_argument("--launches", type=int, default=2)
    a = ap.parse_args()

    import torch

    from . import build, pic, workloads as wk
    build.build()
    wl = wk.WORKLOADS[a.workload]
    x = wk.make_inputs(wl, batch=a.images or None)
    B = x.latents.shape[0]
    prec = a.precision or wl.precisions[-1]
    dec = pic.Decoder.for_workload(wl, prec, max_batch=B)
    dev = torch.device("cuda:0")
    lat = torch.from_numpy(x.latents).to(dev)
    st = torch.from_numpy(x.steps).to(dev)
    w = torch.from_numpy(np.ascontiguousarray(x.weights_for(prec))).to(dev)
    out = torch.empty((B, 3, wl.H, wl.W), dtype=torch.float32, device=dev)
    for _ in range(a.launches):
        dec.decode_batch(lat, st, w, wl.H, wl.W, out, B=B)
    dec.check()
    torch.cuda.synchronize()
    print(f"{dec.kernel_name}: {a.launches} launches of {B} x {wl.W}x{wl.H} ok")
    dec.close()


if __name__ == "__main__":
    main()
