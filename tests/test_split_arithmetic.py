"""The operand arithmetic of the tensor-core path, emulated on the CPU (no GPU).

The tensor path multiplies fp16 operands with fp32 accumulation.  Every
activation operand a (features and hidden values, fp32) is split into two fp16
terms, hi = fp16 rounded toward zero of a and lo = fp16 rounded to nearest of
(a - hi); each layer then computes W hi + W lo (the split-operand tensor GEMM
of Markidis et al., 2018).  These tests pin the facts the kernel relies on:

- a - hi is exact in fp32, and lo has the sign of a (or is 0), so ReLU may be
  applied to hi and lo separately (the kernel fuses it into both conversions);
- hi + lo is a to about 22 significant bits;
- on a full 768x512 image of the 64-image workload (7-64-64-3 ReLU, fp16
  weights), the split decode stays far inside the 4e-3 bar against the fp64
  oracle, while plain fp16 operands (one rounding to nearest) do not have
  that margin.

The emulation is numpy in fp64 with explicit fp16 roundings; it is not the
kernel, and the oracle's whole-image decode is the reference.
"""
import numpy as np

from paper_2609_09020_gb300 import workloads as wk


def rz16(a):
    """fp16 rounding toward zero of fp32 values inside the fp16 range: round
    to nearest, then, where that went away from zero, one step back (fp16 is
    sign-magnitude, so that step is one less in the bit pattern).  fp16 to
    fp32 is exact, so the comparison is made in fp32."""
    a = np.asarray(a, dtype=np.float32)
    h = a.astype(np.float16)
    away = np.abs(h.astype(np.float32)) > np.abs(a)
    return (h.view(np.uint16) - away.astype(np.uint16)).view(np.float16)


def split(a32):
    """(hi, lo) as the kernel forms them from fp32 a: hi = RZ16(a); the
    difference a - hi in fp32; lo = RN16 of that difference."""
    hi = rz16(a32)
    r = (a32 - hi.astype(np.float32)).astype(np.float32)
    return hi, r.astype(np.float16)


def _values(seed=0, n=200_000):
    rng = np.random.default_rng(seed)
    mag = 2.0 ** rng.uniform(-26, 15.9, n)
    v = (np.where(rng.random(n) < 0.5, -1.0, 1.0) * mag).astype(np.float32)
    special = np.array([0.0, -0.0, 65504.0, -65504.0, 2.0 ** -14, 2.0 ** -24, 1.0, -1.0,
                        1.0 + 2.0 ** -10, 1.0 + 2.0 ** -11, 1.0 + 2.0 ** -23, 3.0e-8, 0.1, -0.1],
                       dtype=np.float32)
    return np.concatenate([v, special])


def test_rz16_rounds_toward_zero():
    # fp16 neighbours of 1: 1 and 1 + 2^-10; of -3: -3 and -3 - 2^-9
    a = np.array([1.0 + 2.0 ** -11, 1.0 + 2.0 ** -10 - 2.0 ** -20, -(3.0 + 2.0 ** -9 - 2.0 ** -20),
                  2.0 ** -24 * 1.9, 65504.0, 0.0, -0.0], dtype=np.float32)
    want = [1.0, 1.0, -3.0, 2.0 ** -24, 65504.0, 0.0, 0.0]
    assert rz16(a).astype(np.float64).tolist() == want
    v = _values(3)
    h = rz16(v).astype(np.float64)
    # nothing of fp16 lies strictly between h and v
    with np.errstate(over="ignore"):  # the step above 65504 is inf
        nxt = np.nextafter(rz16(v), np.where(v >= 0, np.float16(np.inf), np.float16(-np.inf)))
    assert np.all(np.abs(h) <= np.abs(v.astype(np.float64)))
    fin = np.isfinite(nxt.astype(np.float64))
    assert np.all(np.abs(nxt.astype(np.float64))[fin] > np.abs(v.astype(np.float64))[fin])


def test_difference_is_exact_and_keeps_the_sign():
    a = _values()
    hi, lo = split(a)
    hi64, a64 = hi.astype(np.float64), a.astype(np.float64)
    assert np.all(np.abs(hi64) <= np.abs(a64))
    assert np.all((hi64 == 0) | (np.sign(hi64) == np.sign(a64)))
    # a - hi in fp32 equals the exact difference
    r32 = (a - hi.astype(np.float32)).astype(np.float32).astype(np.float64)
    assert np.array_equal(r32, a64 - hi64)
    lo64 = lo.astype(np.float64)
    assert np.all((lo64 == 0) | (np.sign(lo64) == np.sign(a64)))


def test_relu_applies_to_each_term():
    a = _values(1)
    hi, lo = split(a)
    relu = lambda v: np.maximum(v.astype(np.float64), 0.0)
    assert np.array_equal(relu(hi) + relu(lo), relu(hi.astype(np.float64) + lo.astype(np.float64)))
    # and it equals the split of relu(a): zero for every negative a
    neg = a < 0
    assert np.all(relu(hi)[neg] == 0) and np.all(relu(lo)[neg] == 0)


def test_split_carries_about_22_bits():
    a = _values(2)
    hi, lo = split(a)
    a64 = a.astype(np.float64)
    err = np.abs(a64 - hi.astype(np.float64) - lo.astype(np.float64))
    # RZ leaves |a - hi| below one fp16 ulp of a (2^(e-10)); RN of that to
    # fp16 errs by at most half an fp16 ulp of it: 2^(e-21) <= 2^-21 |a|, or
    # 2^-25 (half the fp16 subnormal spacing) where the difference is subnormal
    assert np.all(err <= np.maximum(2.0 ** -21 * np.abs(a64), 2.0 ** -25))
    # plain fp16 (one rounding to nearest) keeps 11 bits: relative errors
    # reach 2^-12 on these values, against at most 2^-21 for the split
    normal = np.abs(a64) >= 2.0 ** -14
    rel_plain = np.abs(a64 - a.astype(np.float16).astype(np.float64))[normal] / np.abs(a64[normal])
    assert 2.0 ** -13 < rel_plain.max() <= 2.0 ** -11


def _features(orc, x, b):
    """The image's concatenated upsampled features [D][H*W] (fp64, from the
    oracle's upsampling), rounded to fp32 as the kernel holds them."""
    wl = x.wl
    feats, off = [], 0
    for l in range(wl.L):
        h, w = wk.level_size(wl.H, l), wk.level_size(wl.W, l)
        for _c in range(wl.C):
            q = x.latents[b, off:off + h * w].reshape(h, w)
            off += h * w
            feats.append(orc.upsample(q.astype(np.float64) * float(x.steps[b, l]), wl.H, wl.W))
    return np.stack(feats).reshape(len(feats), -1).astype(np.float32)


def _layers(wv, dims):
    out, p = [], 0
    for k in range(len(dims) - 1):
        n = dims[k + 1] * dims[k]
        out.append((wv[p:p + n].reshape(dims[k + 1], dims[k]), wv[p + n:p + n + dims[k + 1]]))
        p += n + dims[k + 1]
    return out


def _emulate(F32, layers, operand):
    """The MLP with each layer's activation operand replaced by operand(h)
    (fp64 values of its fp16 terms); ReLU hidden layers, clamped output."""
    h = F32
    for k, (W, bias) in enumerate(layers):
        z = W @ operand(h) + bias[:, None]
        h = np.maximum(z, 0).astype(np.float32) if k < len(layers) - 1 else z
    return np.clip(h, 0.0, 1.0)


def _split_operand(h):
    hi, lo = split(h.astype(np.float32))
    return hi.astype(np.float64) + lo.astype(np.float64)


def _plain_operand(h):
    return h.astype(np.float32).astype(np.float16).astype(np.float64)


def _max_error(F32, layers, operand, ref, chunk=32768):
    """max |emulated - ref| over all pixels, a chunk of pixels at a time."""
    return max(float(np.abs(_emulate(F32[:, p:p + chunk], layers, operand)
                            - ref[:, p:p + chunk]).max())
               for p in range(0, F32.shape[1], chunk))


def test_split_meets_the_bar_with_margin_on_a_full_image(orc):
    wl = wk.WORKLOADS["c5"]
    assert wl.act == "relu" and wl.dims == (7, 64, 64, 3)
    x = wk.make_inputs(wl, batch=1)
    w16 = x.weights_for("fp16_tc")[0]
    assert w16.dtype == np.float16  # the weights are fp16 by definition: used exactly
    ref = orc.decode(x.latents[0], x.steps[0], x.oracle_weights("fp16_tc")[0], wl.H, wl.W,
                     wl.L, wl.C, wl.dims, wl.act, nthreads=4).reshape(3, -1)
    F = _features(orc, x, 0)
    layers = _layers(w16.astype(np.float64), wl.dims)
    err_split = _max_error(F, layers, _split_operand, ref)
    err_plain = _max_error(F, layers, _plain_operand, ref)
    assert err_split < 2e-5                 # the bar is 4e-3
    assert err_plain > 1e-3                 # plain fp16: within 4x of the bar
    assert err_plain > 100 * err_split


def e4m3(v):
    """Round to nearest even onto the OCP fp8 e4m3 grid (3 mantissa bits,
    normal exponents -6..8, subnormal spacing 2^-9), saturating at 448."""
    v = np.asarray(v, dtype=np.float64)
    a = np.abs(v)
    e = np.clip(np.floor(np.log2(np.maximum(a, 2.0 ** -30))), -6, 8)
    step = 2.0 ** (e - 3)
    return np.sign(v) * np.minimum(np.round(a / step) * step, 448.0)


def test_e4m3_grid():
    got = e4m3(np.array([448.0, 500.0, 1.0625, 1.1875, 2.0 ** -9, 2.0 ** -10 * 1.01, 3.0 * 2.0 ** -9,
                         -0.3]))
    # 1.0625 is halfway between 1 and 1.125 (even: 1); 1.1875 between 1.125
    # and 1.25 (even: 1.25); 0.3 lies between 0.28125 and 0.3125 (nearer 0.3125)
    assert got.tolist() == [448.0, 448.0, 1.0, 1.25, 2.0 ** -9, 2.0 ** -9, 3.0 * 2.0 ** -9, -0.3125]


def _fp8_lo_operand_layers(layers, S=2.0 ** 6):
    """The MLP as a tensor path with the lo term in fp8 would compute it.
    Hidden activations stay scaled by S (ReLU commutes with a positive
    scale): the hidden operand is hi = RZ16(S h) in fp16 against the fp16
    weights W, plus lo = e4m3(S h - hi) against e4m3(W) (S h - hi is about
    2^-11 S h, inside e4m3's range for S = 2^6 (the kernel's), exact in fp32);
    the bias rows carry S b, the first layer's weights S W (exact: S is a
    power of two), and only the 3 outputs are divided by S.  No rescaling
    of the hidden values is needed, so the epilogue keeps its instruction
    count; the lo MMAs take half the K-steps (32 e4m3 per step)."""
    def run(F32):
        h = F32
        for k, (W, bias) in enumerate(layers):
            if k == 0:
                z = S * (W @ _split_operand(h)) + S * bias[:, None]
            else:
                hs = h.astype(np.float32)          # already scaled by S
                assert np.abs(hs).max() < 65504
                hi = rz16(hs)
                lo = (hs - hi.astype(np.float32)).astype(np.float64)
                z = W @ hi.astype(np.float64) + e4m3(W) @ e4m3(lo) + S * bias[:, None]
            h = np.maximum(z, 0).astype(np.float32) if k < len(layers) - 1 else z / S
        return np.clip(h, 0.0, 1.0)
    return run


def test_fp8_lo_term_stays_inside_the_bar(orc):
    """The arithmetic of the tensor path's fp8 lo term (PIC_PREC_FP16_TC_LO8)
    keeps the error near 2e-4 on a full c5 image (2.2e-4), some 20x inside
    the 4e-3 bar and 12x below plain fp16 (over 8 of the 64 images: 3.4e-4)."""
    wl = wk.WORKLOADS["c5"]
    x = wk.make_inputs(wl, batch=1)
    ref = orc.decode(x.latents[0], x.steps[0], x.oracle_weights("fp16_tc")[0], wl.H, wl.W,
                     wl.L, wl.C, wl.dims, wl.act, nthreads=4).reshape(3, -1)
    F = _features(orc, x, 0)
    layers = _layers(x.weights_for("fp16_tc")[0].astype(np.float64), wl.dims)
    run = _fp8_lo_operand_layers(layers)
    err = max(float(np.abs(run(F[:, p:p + 32768]) - ref[:, p:p + 32768]).max())
              for p in range(0, F.shape[1], 32768))
    err_split = _max_error(F, layers, _split_operand, ref)
    err_plain = _max_error(F, layers, _plain_operand, ref)
    assert err_split < err < 4e-4 and 10 * err < err_plain
