"""GPU inverse DCT stage (dequantise, 8x8 iDCT, un-patchify; Sec. 3.2 Eqs.
5-7 run backwards) and the decode from its fp32 latents, against the fp64
oracle, through the C ABI.

Bars:
  * iDCT latents: |GPU - oracle| <= 24 u (|c|^T |S step| |c|)[m][n] per
    element, u = 2^-24 -- the fp32 error bound of the two 8-term passes
    (one rounding of S * step, 8 FMAs per pass, c rounded to fp32), |c| the
    magnitudes of the DCT basis;
  * decode from fp32 latents: the decode's own bars (fp32 path 1e-4, tensor
    path 4e-3 and 0.02 dB) against the oracle decode of the same fp32
    latents;
  * the chained stages (symbols -> iZpR -> iDCT -> decode) against the
    oracle's chain in fp64 from the same symbols, same bars.
"""
import numpy as np
import pytest

from paper_2609_09020_gb300 import workloads as wk

from decode_util import ORACLE_THREADS, TOL, max_abs_diff, psnr

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_09020_gb300 import build
    build.build()


# ---------------------------------------------------------------- helpers
def _abs_basis():
    k = np.arange(8)[:, None]
    n = np.arange(8)[None, :]
    a = np.where(k == 0, np.sqrt(1 / 8), 0.5)
    return np.abs(a * np.cos((2 * n + 1) * k * np.pi / 16))


def _place(blocks, H, W, L, C):
    """Places real 8x8 blocks [n][8][8] (patch order) into the pyramid layout
    (test-side bookkeeping for the per-element tolerance map)."""
    out = np.zeros(wk.latent_count(H, W, L, C))
    b, off = 0, 0
    for l in range(L):
        h, w = wk.level_size(H, l), wk.level_size(W, l)
        for c in range(C):
            g = out[off + c * h * w: off + (c + 1) * h * w].reshape(h, w)
            for by in range((h + 7) // 8):
                for bx in range((w + 7) // 8):
                    r, q = 8 * by, 8 * bx
                    g[r:r + 8, q:q + 8] = blocks[b][: min(8, h - r), : min(8, w - q)]
                    b += 1
        off += C * h * w
    return out


def _tol_map(coeffs, steps, H, W, L, C):
    A = _abs_basis()
    per_lvl = []
    for l in range(L):
        per_lvl += [steps[l]] * (C * ((wk.level_size(H, l) + 7) // 8) *
                                 ((wk.level_size(W, l) + 7) // 8))
    S = np.abs(coeffs.reshape(-1, 8, 8).astype(np.float64)) * np.array(per_lvl)[:, None, None]
    bound = 24 * 2.0 ** -24 * np.einsum("um,buv,vn->bmn", A, S, A)
    return _place(bound, H, W, L, C)


def _gpu_idct(coeffs, steps, H, W, L, C):
    import torch
    from paper_2609_09020_gb300 import pic
    c = torch.from_numpy(np.ascontiguousarray(coeffs, dtype=np.int32)).cuda()
    s = torch.from_numpy(np.ascontiguousarray(steps, dtype=np.float32)).cuda()
    out = pic.idct_unpatchify(c, s, H, W, L, C)
    torch.cuda.synchronize()
    return out.cpu().numpy()


def _gpu_decode_values(wl, lat_f32, weights, precision, clamp=True):
    import torch
    from paper_2609_09020_gb300.pic import Decoder
    B = lat_f32.shape[0]
    dec = Decoder.for_workload(wl, precision, clamp=clamp, max_batch=B, latent="fp32")
    lat = torch.from_numpy(np.ascontiguousarray(lat_f32, dtype=np.float32)).cuda()
    wt = torch.from_numpy(np.ascontiguousarray(weights)).cuda()
    out = torch.full((B, 3, wl.H, wl.W), float("nan"), dtype=torch.float32, device="cuda")
    dec.decode_batch(lat, None, wt, wl.H, wl.W, out, B=B)
    dec.check()
    torch.cuda.synchronize()
    name = dec.kernel_name
    dec.close()
    return out.cpu().numpy(), name


def _noisy_target(ref, seed):
    rng = np.random.Generator(np.random.PCG64(seed))
    return np.clip(ref + rng.normal(0.0, 10 ** (-35 / 20), ref.shape), 0.0, 1.0)


def _check_rgb(got, want, precision, tag):
    d, where = max_abs_diff(got, want)
    assert d <= TOL[precision], (tag, d, where)
    if precision == "fp16_tc":
        t = _noisy_target(want, 77)
        assert abs(psnr(got, t) - psnr(want, t)) <= 0.02, tag
    return d


# ------------------------------------------------------- the iDCT stage
@pytest.mark.parametrize("H,W,L,C,B", [
    (256, 256, 4, 1, 1),      # whole 8x8 patches everywhere
    (67, 45, 4, 2, 2),        # ragged patches on every level, 2 channels
    (13, 200, 3, 3, 1),       # 3 channels, one ragged patch row
    (8, 8, 1, 1, 3),          # one patch per image
    (1, 1, 1, 1, 2),          # a single latent per image
    (5, 3, 4, 4, 1),          # 4 channels, every level a single ragged patch
])
def test_idct_matches_oracle(orc, H, W, L, C, B):
    rng = np.random.Generator(np.random.PCG64(H * 1000 + W))
    n = wk.block_count(H, W, L, C)
    coeffs = rng.integers(-255, 256, (B, n, 64)).astype(np.int32)
    coeffs[rng.random(coeffs.shape) < 0.5] = 0
    steps = np.array([[1.0, 0.5, 0.3, 0.125][:L]] * B, dtype=np.float32)
    steps[-1, 0] = 0.7
    got = _gpu_idct(coeffs, steps, H, W, L, C)
    assert got.shape == (B, wk.latent_count(H, W, L, C))
    for b in range(B):
        st = steps[b].astype(np.float64)
        want = orc.unpatchify_idct(coeffs[b], st, H, W, L, C)
        tol = _tol_map(coeffs[b], st, H, W, L, C)
        assert np.all(np.abs(got[b] - want) <= tol + 1e-30), (H, W, L, C, b)


def test_idct_full_batch_sampled(orc):
    """The 64-image batch's coefficients (8,192 patches per 768x512 pyramid)
    in one launch; images 0, 31 and 63 checked element by element."""
    x = wk.make_dct_inputs("c5")
    wl = x.wl
    got = _gpu_idct(x.coeffs, x.steps, wl.H, wl.W, wl.L, wl.C)
    for b in (0, 31, 63):
        st = x.steps[b].astype(np.float64)
        want = orc.unpatchify_idct(x.coeffs[b], st, wl.H, wl.W, wl.L, wl.C)
        tol = _tol_map(x.coeffs[b], st, wl.H, wl.W, wl.L, wl.C)
        assert np.all(np.abs(got[b] - want) <= tol + 1e-30), b


# ------------------------------------- decode from fp32 latents (every arch)
def _arch_case(name):
    """The decode workloads' architectures on sizes the oracle decodes in
    seconds (c3/c4 architectures on reduced, ragged images)."""
    base = wk.WORKLOADS[name]
    size = {"c1": (256, 256), "c2": (512, 768), "c3": (270, 482), "c4": (131, 517),
            "c5": (512, 768)}[name]
    return base.replace(H=size[0], W=size[1], seeds=base.seeds[:2])


@pytest.mark.parametrize("name", ["c1", "c2", "c3", "c4", "c5"])
@pytest.mark.parametrize("precision", ["fp32", "fp16_tc"])
def test_decode_fp32_latents(orc, name, precision):
    wl = _arch_case(name)
    x = wk.make_dct_inputs(wl)
    B = x.coeffs.shape[0]
    lat = np.stack([orc.unpatchify_idct(x.coeffs[b], x.steps[b].astype(np.float64), wl.H, wl.W,
                                        wl.L, wl.C) for b in range(B)]).astype(np.float32)
    w = x.weights_for(precision)
    got, kname = _gpu_decode_values(wl, lat, w, precision)
    assert kname.endswith("_f32lat"), kname
    if precision == "fp16_tc":
        assert kname.startswith("tc05_"), kname
    for b in range(B):
        want = orc.decode_values(lat[b].astype(np.float64), w[b].astype(np.float64), wl.H, wl.W,
                                 wl.L, wl.C, wl.dims, wl.act, nthreads=ORACLE_THREADS)
        _check_rgb(got[b], want, precision, (name, precision, b))


def test_decode_fp32_latents_generic_and_raw(orc):
    """An architecture without a specialisation (generic fp32 kernel) and
    the unclamped output."""
    wl = wk.custom("g", H=37, W=61, L=3, C=2, dims=(6, 20, 12, 3), act="gelu", batch=2)
    x = wk.make_dct_inputs(wl)
    lat = np.stack([orc.unpatchify_idct(x.coeffs[b], x.steps[b].astype(np.float64), wl.H, wl.W,
                                        wl.L, wl.C) for b in range(2)]).astype(np.float32)
    got, kname = _gpu_decode_values(wl, lat, x.weights_for("fp32"), "fp32", clamp=False)
    assert kname == "fp32_generic_f32lat"
    for b in range(2):
        want = orc.decode_values(lat[b].astype(np.float64), x.weights[b].astype(np.float64),
                                 wl.H, wl.W, wl.L, wl.C, wl.dims, wl.act, clamp=False)
        d, where = max_abs_diff(got[b], want)
        assert d <= 1e-4 * max(1.0, float(np.abs(want).max())), (b, d, where)


# ----------------------------------------------------------- chained stages
@pytest.mark.parametrize("precision", ["fp32", "fp16_tc"])
def test_chain_idct_then_decode(orc, precision):
    """Coefficients -> GPU iDCT -> GPU decode, against the oracle's fp64 chain
    (no fp32 rounding of the latents on the oracle side)."""
    import torch
    from paper_2609_09020_gb300 import pic
    wl = _arch_case("c5")
    x = wk.make_dct_inputs(wl)
    B = x.coeffs.shape[0]
    c = torch.from_numpy(x.coeffs).cuda()
    s = torch.from_numpy(x.steps).cuda()
    lat = pic.idct_unpatchify(c, s, wl.H, wl.W, wl.L, wl.C)
    dec = pic.Decoder.for_workload(wl, precision, max_batch=B, latent="fp32")
    w = x.weights_for(precision)
    out = torch.empty((B, 3, wl.H, wl.W), dtype=torch.float32, device="cuda")
    dec.decode_batch(lat, None, torch.from_numpy(np.ascontiguousarray(w)).cuda(), wl.H, wl.W,
                     out, B=B)
    dec.check()
    got = out.cpu().numpy()
    dec.close()
    for b in range(B):
        y = orc.unpatchify_idct(x.coeffs[b], x.steps[b].astype(np.float64), wl.H, wl.W, wl.L, wl.C)
        want = orc.decode_values(y, w[b].astype(np.float64), wl.H, wl.W, wl.L, wl.C, wl.dims,
                                 wl.act, nthreads=ORACLE_THREADS)
        _check_rgb(got[b], want, precision, ("chain", precision, b))


def test_chain_from_zpr_symbols(orc):
    """ZpR symbol stream -> GPU iZpR (Algorithm 1) -> GPU iDCT -> GPU decode:
    the decoder after entropy decoding, against the oracle's chain."""
    import torch
    from paper_2609_09020_gb300 import pic
    wl = wk.WORKLOADS["c1"]
    x = wk.make_dct_inputs(wl)
    n_blk = x.coeffs.shape[1]
    eob = wk.DCT_CLIP + 17
    stream = orc.zpr_encode(x.coeffs[0], eob)
    sym = torch.from_numpy(stream).cuda()
    coeffs, offsets = pic.izpr_decode(sym, eob, n_blk)
    lat = pic.idct_unpatchify(coeffs, torch.from_numpy(x.steps).cuda(), wl.H, wl.W, wl.L, wl.C)
    dec = pic.Decoder.for_workload(wl, "fp32", max_batch=1, latent="fp32")
    out = torch.empty((1, 3, wl.H, wl.W), dtype=torch.float32, device="cuda")
    dec.decode_batch(lat, None, torch.from_numpy(x.weights_for("fp32")).cuda(), wl.H, wl.W, out,
                     B=1)
    dec.check()
    got = out.cpu().numpy()[0]
    dec.close()
    assert np.array_equal(coeffs.cpu().numpy(), orc.izpr(stream, eob, n_blk))
    y = orc.unpatchify_idct(orc.izpr(stream, eob, n_blk), x.steps[0].astype(np.float64), wl.H,
                            wl.W, wl.L, wl.C)
    want = orc.decode_values(y, x.weights[0].astype(np.float64), wl.H, wl.W, wl.L, wl.C,
                             wl.dims, wl.act)
    _check_rgb(got, want, "fp32", "zpr chain")
