"""GPU modulation fusion (App. A) against the fp64 oracle, through the C ABI:
the fused weight blobs element by element, and whole decodes with the fused
weights against the oracle's un-fused decode (MLP^s -> normalise ->
modulate -> MLP^i)."""
import numpy as np
import pytest

from paper_2609_09020_gb300 import workloads as wk

from decode_util import ORACLE_THREADS, TOL, max_abs_diff, psnr

pytestmark = pytest.mark.gpu
U = 2.0 ** -24


@pytest.fixture(scope="module", autouse=True)
def _built():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_09020_gb300 import build
    build.build()


def _last_layer(dims):
    off = sum(dims[k + 1] * (dims[k] + 1) for k in range(len(dims) - 2))
    return off, dims[-2]


def _gpu_fuse(dims, precision, shared, mod):
    import torch
    from paper_2609_09020_gb300 import pic
    L = dims[0]
    arch = pic.make_arch(L, 1, dims, "relu", precision, max_H=8, max_W=8)
    out = pic.fuse_modulation(arch, torch.from_numpy(shared).cuda(), torch.from_numpy(mod).cuda())
    torch.cuda.synchronize()
    return out.cpu().numpy()


@pytest.mark.parametrize("precision", ["fp32", "fp16_tc"])
@pytest.mark.parametrize("dims", [(7, 64, 64, 3), (16, 64, 64, 64, 3), (4, 16, 3)])
def test_fused_blob_matches_oracle(orc, dims, precision):
    dims = list(dims)
    rng = np.random.Generator(np.random.PCG64(len(dims) * 100 + dims[1]))
    P = orc.param_count(dims)
    shared = rng.normal(0, 0.3, P).astype(np.float32)
    off, cf = _last_layer(dims)
    mod = wk.make_modulation(5, cf, 3)
    got = _gpu_fuse(dims, precision, shared, mod).astype(np.float64)
    w = shared[off:off + 3 * cf].astype(np.float64).reshape(3, cf)
    b = shared[off + 3 * cf:].astype(np.float64)
    for i in range(5):
        g, be, mu, sd = mod[i].astype(np.float64)
        wf, bf = orc.fuse_modulation(w, b, g, be, mu, sd)
        want = np.concatenate([shared[:off].astype(np.float64), wf.ravel(), bf])
        # error bounds of the fp32 arithmetic (products/quotients: 3 roundings;
        # the bias: a sum of cf terms, each with 4 roundings)
        tol = np.zeros(P)
        tol[off:off + 3 * cf] = 4 * U * np.abs(wf.ravel())
        tol[off + 3 * cf:] = (cf + 6) * U * (np.abs(b) + np.abs(w) @ (np.abs(be) + 2 * np.abs(g * mu / sd)))
        if precision == "fp32":
            assert np.array_equal(got[i, :off], want[:off])            # copied exactly
            assert np.all(np.abs(got[i] - want) <= tol), i
        else:
            # the blob is the fp16 rounding (to nearest) of the fp32 result
            assert np.array_equal(got[i, :off], shared[:off].astype(np.float16).astype(np.float64))
            assert np.all(np.abs(got[i] - want) <= tol + 2.0 ** -11 * np.abs(want) + 2.0 ** -25), i


def _case():
    return wk.custom("fuse", H=120, W=184, L=7, C=1, dims=(7, 64, 64, 3), act="relu", batch=2,
                     seed=40)


def test_fused_decode_equals_unfused_oracle_fp32(orc):
    """GPU fusion + GPU decode (fp32 path) against the oracle's un-fused
    decode with each image's own statistics."""
    import torch
    from paper_2609_09020_gb300 import pic
    wl = _case()
    x = wk.make_inputs(wl)
    shared = x.weights[0].astype(np.float32)
    off, cf = _last_layer(list(wl.dims))
    mod = wk.make_modulation(wl.B, cf, 5)
    for b in range(wl.B):  # the image's own MLP^s statistics
        mu, sd = orc.mlps_stats(x.latents[b], x.steps[b].astype(np.float64), shared.astype(np.float64),
                                wl.H, wl.W, wl.L, wl.C, wl.dims, wl.act)
        mod[b, 2], mod[b, 3] = mu, sd
    dec = pic.Decoder.for_workload(wl, "fp32", max_batch=wl.B)
    wts = pic.fuse_modulation(dec.arch, torch.from_numpy(shared).cuda(), torch.from_numpy(mod).cuda())
    out = torch.empty((wl.B, 3, wl.H, wl.W), dtype=torch.float32, device="cuda")
    dec.decode_batch(torch.from_numpy(x.latents).cuda(), torch.from_numpy(x.steps).cuda(), wts, wl.H,
                     wl.W, out, B=wl.B)
    dec.check()
    got = out.cpu().numpy()
    dec.close()
    for b in range(wl.B):
        g, be, mu, sd = mod[b].astype(np.float64)
        want = orc.decode_modulated(x.latents[b], x.steps[b].astype(np.float64),
                                    shared.astype(np.float64), wl.H, wl.W, wl.L, wl.C, wl.dims,
                                    wl.act, g, be, mu, sd, nthreads=ORACLE_THREADS)
        d, where = max_abs_diff(got[b], want)
        assert d <= TOL["fp32"], (b, d, where)
        assert 0.05 < float(((want > 0) & (want < 1)).mean())  # not all clamped


def test_fused_decode_tensor_path(orc):
    """GPU fusion to fp16 + the tensor-core decode against the oracle decode
    of the same fp16 blob (the path's input), with the decode's bars."""
    import torch
    from paper_2609_09020_gb300 import pic
    wl = _case()
    x = wk.make_inputs(wl)
    shared = x.weights[0].astype(np.float32)
    off, cf = _last_layer(list(wl.dims))
    mod = wk.make_modulation(wl.B, cf, 6)
    dec = pic.Decoder.for_workload(wl, "fp16_tc", max_batch=wl.B)
    wts = pic.fuse_modulation(dec.arch, torch.from_numpy(shared).cuda(), torch.from_numpy(mod).cuda())
    out = torch.empty((wl.B, 3, wl.H, wl.W), dtype=torch.float32, device="cuda")
    dec.decode_batch(torch.from_numpy(x.latents).cuda(), torch.from_numpy(x.steps).cuda(), wts, wl.H,
                     wl.W, out, B=wl.B)
    dec.check()
    got, blob = out.cpu().numpy(), wts.cpu().numpy().astype(np.float64)
    dec.close()
    rng = np.random.Generator(np.random.PCG64(9))
    for b in range(wl.B):
        want = orc.decode(x.latents[b], x.steps[b].astype(np.float64), blob[b], wl.H, wl.W, wl.L,
                          wl.C, wl.dims, wl.act, nthreads=ORACLE_THREADS)
        d, where = max_abs_diff(got[b], want)
        assert d <= TOL["fp16_tc"], (b, d, where)
        t = np.clip(want + rng.normal(0, 10 ** (-35 / 20), want.shape), 0, 1)
        assert abs(psnr(got[b], t) - psnr(want, t)) <= 0.02
