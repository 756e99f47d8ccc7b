"""Pins of the fp64 oracle: facts fixed by the paper's definitions and by
mathematics, independent of the oracle's own code.

Each pin takes an ``oracle.Oracle`` and raises AssertionError when the oracle
disagrees.  ``test_oracle.py`` runs every pin on the real oracle;
``test_oracle_mutations.py`` runs them on copies of the oracle with a planted
mistake and requires every planted mistake to fail at least one pin.
"""
from __future__ import annotations

import math
import os
from fractions import Fraction

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _frac(tok: str) -> float:
    return float(Fraction(tok))


def load_golden(name: str) -> dict:
    out = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            key, *vals = line.split()
            out[key] = vals
    return out


# ---------------------------------------------------------------- shapes
def pin_level_sizes(o):
    """Eq. 1 with the ceiling reading: H_l = ceil(H / 2^l)."""
    assert [o.level_size(1080, l) for l in range(7)] == [1080, 540, 270, 135, 68, 34, 17]
    assert [o.level_size(1920, l) for l in range(7)] == [1920, 960, 480, 240, 120, 60, 30]
    assert [o.level_size(768, l) for l in range(7)] == [768, 384, 192, 96, 48, 24, 12]
    assert [o.level_size(5, l) for l in range(4)] == [5, 3, 2, 1]
    assert o.latent_count(256, 256, 4, 1) == 256 ** 2 + 128 ** 2 + 64 ** 2 + 32 ** 2
    assert o.latent_count(5, 3, 3, 2) == 2 * (15 + 6 + 2)
    assert o.param_count([4, 16, 16, 3]) == 16 * 5 + 16 * 17 + 3 * 17


# ---------------------------------------------------------------- dequant
def pin_dequant_exact(o):
    """y = q * step; with step = 2^-l every product is an exact dyadic."""
    q = np.arange(-63, 64, dtype=np.int32)
    for l in range(8):
        y = o.dequant(q, 2.0 ** -l)
        assert np.array_equal(y, q.astype(np.float64) / (1 << l))
    y = o.dequant(np.array([3, -5], dtype=np.int32), 0.3)
    assert y[0] == 3 * 0.3 and y[1] == -5 * 0.3


# ---------------------------------------------------------------- upsampling
def _src_coord(x: int, n_in: int, n_out: int) -> Fraction:
    """Half-pixel-centre source coordinate, exact, clamped to [0, n_in - 1]."""
    s = (Fraction(2 * x + 1) * n_in) / (2 * n_out) - Fraction(1, 2)
    return min(max(s, Fraction(0)), Fraction(n_in - 1))


def pin_upsample_constant(o):
    """A constant grid upsamples to the same constant everywhere."""
    for (hl, wl, H, W) in [(1, 1, 7, 5), (2, 3, 4, 6), (17, 30, 135, 240), (3, 2, 5, 3)]:
        g = np.full((hl, wl), -2.75)
        out = o.upsample(g, H, W)
        assert np.array_equal(out, np.full((H, W), -2.75))


def pin_upsample_affine(o):
    """Bilinear interpolation reproduces an affine grid a + b u + c v exactly,
    at the (clamped) source coordinate of every output pixel.  Dyadic values
    and power-of-two scales keep every fp64 operation exact."""
    a, b, c = 1.5, 0.25, -2.0
    for (hl, wl, H, W) in [(8, 4, 32, 16), (2, 2, 4, 4), (4, 8, 32, 64), (1, 4, 8, 16)]:
        v, u = np.mgrid[0:hl, 0:wl]
        g = a + b * u + c * v
        out = o.upsample(g, H, W)
        for y in range(H):
            sy = float(_src_coord(y, hl, H))
            for x in range(W):
                sx = float(_src_coord(x, wl, W))
                assert out[y, x] == a + b * sx + c * sy, (hl, wl, H, W, x, y)


def pin_upsample_separable_bruteforce(o):
    """Bilinear upsampling of an outer product is the outer product of the two
    1-D linear interpolations; each 1-D weight is the tent (1 - |s - u|)^+ at
    the exact rational source coordinate, written out here by brute force.
    Covers ceil-sized (non power-of-two) ratios."""
    rng = np.random.Generator(np.random.PCG64(7))
    for (hl, wl, H, W) in [(3, 5, 5, 9), (17, 30, 135, 240), (2, 1, 3, 1), (34, 60, 270, 480),
                           (1, 2, 1, 3), (68, 120, 1080, 1920)]:
        r = rng.integers(-31, 32, hl).astype(np.float64)
        cvec = rng.integers(-31, 32, wl).astype(np.float64)
        g = np.outer(r, cvec)

        def interp_1d(vals, n_in, n_out, x):
            s = _src_coord(x, n_in, n_out)
            return sum(float(max(Fraction(0), 1 - abs(s - u))) * vals[u] for u in range(n_in))

        ys = np.unique(np.linspace(0, H - 1, min(H, 24)).astype(int))
        xs = np.unique(np.linspace(0, W - 1, min(W, 24)).astype(int))
        ry = {int(y): interp_1d(r, hl, H, int(y)) for y in ys}
        cx = {int(x): interp_1d(cvec, wl, W, int(x)) for x in xs}
        for y in ys:
            for x in xs:
                got = o.bilinear_at(g, H, W, int(x), int(y))
                want = ry[int(y)] * cx[int(x)]
                assert abs(got - want) <= 1e-12 * (1 + abs(want)), (hl, wl, H, W, x, y, got, want)
        full = o.upsample(g, H, W)
        assert np.array_equal(full[ys][:, xs], np.array([[o.bilinear_at(g, H, W, int(x), int(y))
                                                          for x in xs] for y in ys]))


def pin_upsample_identity_scale(o):
    """Level 0 (scale 1) is the identity."""
    rng = np.random.Generator(np.random.PCG64(3))
    g = rng.standard_normal((7, 11))
    assert np.array_equal(o.upsample(g, 7, 11), g)


def pin_upsample_factor2_weights(o):
    """2x upsampling with half-pixel centres uses the weights 3/4, 1/4: output
    column 2u+1 = 3/4 g[u] + 1/4 g[u+1], column 2u+2 = 1/4 g[u] + 3/4 g[u+1]."""
    g = np.array([[1.0, 5.0, -3.0, 8.0]])
    out = o.upsample(g, 1, 8)[0]
    want = [1.0, 0.75 * 1 + 0.25 * 5, 0.25 * 1 + 0.75 * 5, 0.75 * 5 + 0.25 * -3,
            0.25 * 5 + 0.75 * -3, 0.75 * -3 + 0.25 * 8, 0.25 * -3 + 0.75 * 8, 8.0]
    assert np.array_equal(out, np.array(want))
    col = o.upsample(g.T.copy(), 8, 1)[:, 0]
    assert np.array_equal(col, np.array(want))


# ---------------------------------------------------------------- MLP
def pin_act_closed_forms(o):
    """ReLU(z) = max(z, 0).  GELU(z) = z Phi(z): GELU(0) = 0, GELU(1) = Phi(1),
    GELU(z) - GELU(-z) = z (since Phi(z) + Phi(-z) = 1), GELU(z) -> z, 0 at
    +-infinity, and the textbook value Phi(1) = 0.8413447460685429..."""
    assert o.act(0.0, "relu") == 0.0 and o.act(-3.5, "relu") == 0.0 and o.act(2.25, "relu") == 2.25
    assert o.act(0.0, "gelu") == 0.0
    assert abs(o.act(1.0, "gelu") - 0.8413447460685429) < 1e-15
    assert abs(o.act(-1.0, "gelu") - (0.8413447460685429 - 1.0)) < 1e-15
    for z in [0.1, 0.5, 1.7, 3.0, 6.0]:
        assert abs(o.act(z, "gelu") - o.act(-z, "gelu") - z) < 1e-14
    assert abs(o.act(12.0, "gelu") - 12.0) < 1e-20
    assert abs(o.act(-12.0, "gelu")) < 1e-20
    # Phi(2) = 0.9772498680518208 (standard normal table value)
    assert abs(o.act(2.0, "gelu") - 2 * 0.9772498680518208) < 1e-14


def pin_mlp_zero_weights(o):
    """All weights zero: the output is the last bias, whatever the input."""
    dims = [5, 8, 3]
    w = np.zeros(8 * 5 + 8 + 3 * 8 + 3)
    w[-3:] = [0.25, -1.5, 7.0]
    for act in ("relu", "gelu"):
        out = o.mlp(np.array([1.0, -2, 3, -4, 5]), w, dims, act)
        assert np.array_equal(out, np.array([0.25, -1.5, 7.0]))


def _blob(layers):
    return np.concatenate([np.concatenate([np.asarray(Wm, float).ravel(), np.asarray(b, float)])
                           for Wm, b in layers])


def pin_mlp_hand(o):
    """A two-layer MLP worked by hand; exposes transposed weights, dropped or
    misplaced biases, and an activation on the output layer."""
    W0 = [[1.0, 2.0, 0.0], [0.0, -1.0, 1.0]]          # 3 -> 2
    b0 = [0.5, -4.0]
    W1 = [[2.0, 0.0], [1.0, 1.0], [0.0, -3.0]]         # 2 -> 3
    b1 = [0.0, -10.0, 1.0]
    x = np.array([1.0, 2.0, 3.0])
    # z0 = (1 + 4 + 0 + 0.5, 0 - 2 + 3 - 4) = (5.5, -3); relu -> (5.5, 0)
    # out = (11, 5.5 - 10, 0 + 1) = (11, -4.5, 1)
    out = o.mlp(x, _blob([(W0, b0), (W1, b1)]), [3, 2, 3], "relu")
    assert np.array_equal(out, np.array([11.0, -4.5, 1.0]))
    # GELU hidden: h = (5.5 Phi(5.5), -3 Phi(-3))
    phi = lambda z: 0.5 * (1 + math.erf(z / math.sqrt(2)))
    h = [5.5 * phi(5.5), -3 * phi(-3)]
    want = [2 * h[0], h[0] + h[1] - 10, -3 * h[1] + 1]
    out = o.mlp(x, _blob([(W0, b0), (W1, b1)]), [3, 2, 3], "gelu")
    assert np.allclose(out, want, rtol=0, atol=1e-13)


def pin_mlp_identity(o):
    """Identity hidden layers with ReLU pass the positive part through."""
    n = 6
    eye = np.eye(n)
    Wout = np.zeros((3, n))
    Wout[0, 0], Wout[1, 3], Wout[2, 5] = 1.0, 2.0, -1.0
    w = _blob([(eye, np.zeros(n)), (eye, np.zeros(n)), (Wout, [0.0, 0.0, 0.5])])
    x = np.array([1.5, -2.0, 3.0, 0.25, -1.0, -4.0])
    out = o.mlp(x, w, [n, n, n, 3], "relu")
    assert np.array_equal(out, np.array([1.5, 0.5, 0.5]))


def pin_mlp_random_matmul(o):
    """Against independent fp64 matrix products (numpy) on random weights."""
    rng = np.random.Generator(np.random.PCG64(11))
    dims = [7, 40, 40, 3]
    layers = [(rng.standard_normal((dims[k + 1], dims[k])), rng.standard_normal(dims[k + 1]))
              for k in range(3)]
    x = rng.standard_normal(7) * 3
    h = x
    for k, (Wm, b) in enumerate(layers):
        z = Wm @ h + b
        h = z if k == 2 else np.maximum(z, 0)
    out = o.mlp(x, _blob(layers), dims, "relu")
    assert np.allclose(out, h, rtol=1e-13, atol=1e-13)


def pin_clamp(o):
    assert o.clamp01(-0.5) == 0.0 and o.clamp01(1.5) == 1.0 and o.clamp01(0.375) == 0.375


# ---------------------------------------------------------------- decode
def pin_to_u8(o):
    """round-half-even(255 clamp(v)): 0.25 -> 63.75 -> 64, 0.75 -> 191.25 ->
    191, 0.5 -> 127.5 -> 128 (the even neighbour), saturation at both ends."""
    for v, want in ((0.0, 0), (1.0, 255), (-3.0, 0), (7.0, 255), (0.25, 64), (0.75, 191),
                    (0.5, 128), (1.0 / 255.0, 1), (254.4 / 255.0, 254)):
        assert o.to_u8(v) == want, (v, o.to_u8(v), want)


def pin_decode_hand_4x4(o):
    """The hand-computed 4x4 image (tests/golden/hand_4x4.txt)."""
    g = load_golden("hand_4x4.txt")
    H, W, L, C = int(g["H"][0]), int(g["W"][0]), int(g["L"][0]), int(g["C"][0])
    dims = [int(v) for v in g["dims"]]
    lat = np.array([int(v) for v in g["latents_l0"] + g["latents_l1"]], dtype=np.int32)
    steps = np.array([_frac(v) for v in g["steps"]])
    w = np.array([_frac(v) for v in g["weights"]])
    out = o.decode(lat, steps, w, H, W, L, C, dims, g["act"][0], clamp=True)
    for c, key in enumerate("RGB"):
        want = np.array([_frac(v) for v in g[key]]).reshape(H, W)
        assert np.allclose(out[c], want, rtol=0, atol=1e-15), (key, out[c], want)
    # the upsampled level-1 plane, through the upsampler alone
    y1 = o.dequant(np.array([int(v) for v in g["latents_l1"]], dtype=np.int32), steps[1])
    u1 = o.upsample(y1.reshape(2, 2), H, W)
    assert np.array_equal(u1, np.array([_frac(v) for v in g["U1"]]).reshape(H, W))
    # unclamped: B at (3, 3) is 1 - 6/4 = -1/2
    raw = o.decode(lat, steps, w, H, W, L, C, dims, "relu", clamp=False)
    assert raw[2, 3, 3] == -0.5 and raw[1, 3, 3] == 1.0


def pin_decode_feature_order(o):
    """The feature is level-major (finest first), channel-minor: a first layer
    that selects feature index j reproduces exactly level l = j // C, channel
    c = j % C, upsampled."""
    rng = np.random.Generator(np.random.PCG64(5))
    H, W, L, C = 9, 7, 3, 2
    shapes = [((H + (1 << l) - 1) >> l, (W + (1 << l) - 1) >> l) for l in range(L)]
    planes = [rng.integers(-9, 10, (h, w)).astype(np.int32) for (h, w) in shapes for _ in range(C)]
    lat = np.concatenate([p.ravel() for p in planes])
    steps = np.array([1.0, 0.5, 0.25])
    D = L * C
    for j in range(D):
        W0 = np.zeros((3, D))
        W0[0, j] = 1.0
        W0[1, j] = -1.0
        W0[2, (j + 1) % D] = 0.5
        w = np.concatenate([W0.ravel(), np.zeros(3)])
        out = o.decode(lat, steps, w, H, W, L, C, [D, 3], "relu", clamp=False)
        l, c = divmod(j, C)
        want = o.upsample(planes[j].astype(np.float64) * steps[l], H, W)
        assert np.array_equal(out[0], want) and np.array_equal(out[1], -want)
        l2, _ = divmod((j + 1) % D, C)
        want2 = o.upsample(planes[(j + 1) % D].astype(np.float64) * steps[l2], H, W) * 0.5
        assert np.array_equal(out[2], want2)


def pin_decode_single_level(o):
    """L = 1: no interpolation; out = clamp(W1 relu(W0 q s + b0) + b1) per pixel,
    against numpy matrix products."""
    rng = np.random.Generator(np.random.PCG64(9))
    H, W = 6, 5
    q = rng.integers(-15, 16, (1, H, W)).astype(np.int32)
    W0, b0 = rng.standard_normal((4, 1)), rng.standard_normal(4)
    W1, b1 = rng.standard_normal((3, 4)) * 0.3, rng.standard_normal(3) * 0.3 + 0.5
    out = o.decode(q.ravel(), [0.125], _blob([(W0, b0), (W1, b1)]), H, W, 1, 1, [1, 4, 3], "relu")
    f = q.reshape(1, -1).astype(np.float64) * 0.125
    want = np.clip(W1 @ np.maximum(W0 @ f + b0[:, None], 0) + b1[:, None], 0, 1).reshape(3, H, W)
    assert np.allclose(out, want, rtol=0, atol=1e-14)


def pin_decode_pixels_match(o):
    """decode_pixels returns the same values as the full decode at those pixels."""
    rng = np.random.Generator(np.random.PCG64(21))
    H, W, L, C = 13, 10, 3, 1
    n = sum(((H + (1 << l) - 1) >> l) * ((W + (1 << l) - 1) >> l) for l in range(L))
    lat = rng.integers(-31, 32, n).astype(np.int32)
    dims = [3, 8, 3]
    w = rng.standard_normal(8 * 3 + 8 + 3 * 8 + 3) * 0.4
    full = o.decode(lat, [1, .5, .25], w, H, W, L, C, dims, "gelu")
    pix = np.array([0, 9, 55, 129, 64], dtype=np.int64)
    part = o.decode_pixels(lat, [1, .5, .25], w, H, W, L, C, dims, "gelu", pix)
    assert np.array_equal(part, full.reshape(3, -1)[:, pix].T)


# ---------------------------------------------------------------- ZpR (Sec. 3.3, Alg. 1)
def _golden_blocks(g):
    n = int(g["nblocks"][0])
    blocks = np.zeros((n, 64), dtype=np.int32)
    for b in range(n):
        for tok in g.get(f"block{b}", []):
            pos, val = tok.split(":")
            blocks[b, int(pos)] = int(val)
    return blocks


def pin_zigzag_order(o):
    """The zigzag order is a permutation of 0..63 that walks the
    anti-diagonals row + col = 0..14 in turn, alternating direction, starting
    0, 1, 8, 16, 9, 2, 3, 10, 17, 24 (the JPEG order) and ending at 63."""
    z = o.zigzag()
    assert sorted(z.tolist()) == list(range(64))
    assert z[:10].tolist() == [0, 1, 8, 16, 9, 2, 3, 10, 17, 24]
    assert z[-3:].tolist() == [55, 62, 63]
    diag = [int(r // 8 + r % 8) for r in z]
    assert diag == sorted(diag)


def pin_zpr_hand_stream(o):
    """The hand-worked stream of tests/golden/zpr_blocks.txt, both ways."""
    g = load_golden("zpr_blocks.txt")
    eob = int(g["eob"][0])
    blocks = _golden_blocks(g)
    stream = np.array([int(v) for v in g["stream"]], dtype=np.int32)
    assert np.array_equal(o.zpr_encode(blocks, eob), stream)
    assert np.array_equal(o.izpr(stream, eob, blocks.shape[0]), blocks)


def pin_zpr_round_trip(o):
    """Inverse ZpR undoes ZpR on random sparse blocks, all-zero blocks, dense
    blocks and long zero runs (> 16, split over several codes)."""
    rng = np.random.Generator(np.random.PCG64(31))
    b = rng.integers(-20, 21, (200, 64)).astype(np.int32)
    b[rng.random((200, 64)) < 0.8] = 0
    b[5] = 0
    b[6] = rng.integers(1, 9, 64)
    b[7] = 0
    b[7, 63] = -3
    b[8] = 0
    b[8, 0] = 4
    b[8, 62] = 2
    eob = int(np.abs(b).max()) + 17
    s = o.zpr_encode(b, eob)
    assert (s == eob).sum() == 200
    assert np.array_equal(o.izpr(s, eob, 200), b)
    # trailing zeros are trimmed: an all-zero block is the marker alone
    z = o.zpr_encode(np.zeros((3, 64), np.int32), 40)
    assert z.tolist() == [40, 40, 40]


def pin_izpr_rejects_malformed(o):
    """A block longer than 64 positions, or the wrong number of markers, is
    refused."""
    eob = 30
    over = np.array([29, 29, 29, 29, 29, 30], dtype=np.int32)  # 80 zeros
    for s, n in [(over, 1), (np.array([1, 30, 2, 30], dtype=np.int32), 3),
                 (np.array([1, 30, 2, 30], dtype=np.int32), 1)]:
        try:
            o.izpr(s, eob, n)
        except ValueError:
            continue
        raise AssertionError(f"malformed stream accepted: {s.tolist()} n={n}")


# ------------------------------------------- patchify + DCT (Sec. 3.2, Eqs. 5-7)
def pin_dct_matches_scipy(o):
    """The orthonormal 8x8 DCT-II and its inverse are scipy's dctn / idctn
    with norm="ortho" (type II / III)."""
    import scipy.fft as F
    rng = np.random.Generator(np.random.PCG64(41))
    for _ in range(4):
        S = rng.normal(0.0, 10.0, (8, 8))
        assert np.abs(o.idct8x8(S) - F.idctn(S, type=2, norm="ortho")).max() < 1e-12
        assert np.abs(o.dct8x8(S) - F.dctn(S, type=2, norm="ortho")).max() < 1e-12


def pin_dct_closed_forms(o):
    """DC only: S[0][0] = 8c gives the constant c.  S[0][4] = 1 (horizontal
    frequency 4 only): cos((2n+1) pi / 4) = +-1/sqrt 2 and a(0) a(4) =
    1/(4 sqrt 2), so every row is (1, -1, -1, 1, 1, -1, -1, 1) / 8; S[4][0]
    is the same pattern down the columns.  Parseval holds and the two
    transforms invert each other."""
    S = np.zeros((8, 8))
    S[0, 0] = 8 * 2.5
    assert np.abs(o.idct8x8(S) - 2.5).max() < 1e-13
    pat = np.array([1, -1, -1, 1, 1, -1, -1, 1]) / 8.0
    S = np.zeros((8, 8))
    S[0, 4] = 1.0
    assert np.abs(o.idct8x8(S) - pat[None, :]).max() < 1e-14
    S = np.zeros((8, 8))
    S[4, 0] = 1.0
    assert np.abs(o.idct8x8(S) - pat[:, None]).max() < 1e-14
    rng = np.random.Generator(np.random.PCG64(43))
    S = rng.normal(0.0, 5.0, (8, 8))
    x = o.idct8x8(S)
    assert abs((x ** 2).sum() - (S ** 2).sum()) < 1e-10 * (S ** 2).sum()
    assert np.abs(o.dct8x8(x) - S).max() < 1e-12


def pin_block_counts(o):
    """sum_l C ceil(H_l/8) ceil(W_l/8), counted by hand for three pyramids."""
    assert o.block_count(512, 768, 7, 1) == 6144 + 1536 + 384 + 96 + 24 + 6 + 2
    assert o.block_count(256, 256, 4, 1) == 1024 + 256 + 64 + 16
    # 1080 x 1920, 7 levels: 135x240, 68x120, 34x60, 17x30, 9x15, 5x8, 3x4 patches
    assert o.block_count(1080, 1920, 7, 2) == 2 * (32400 + 8160 + 2040 + 510 + 135 + 40 + 12)


def pin_unpatchify_hand(o):
    """A 12 x 10 image, 2 levels, 1 channel, steps (1, 1/2): level 0 has 2 x 2
    patches (the right and bottom ones ragged), level 1 (6 x 5) one.  With
    DC-only patches of DC 8, 16, 24, 32 and 64 the level-0 plane is 1 in the
    top-left 8 x 8, 2 in the top-right 8 x 2, 3 and 4 below; level 1 is
    64 * 1/2 / 8 = 4.  A horizontal-frequency-4 patch in the bottom-left slot
    gives its rows the pattern (1, -1, -1, 1, 1, -1, -1, 1) * S / 8."""
    H, W, L, C = 12, 10, 2, 1
    sym = np.zeros((5, 64), np.int32)
    sym[:, 0] = [8, 16, 24, 32, 64]
    y = o.unpatchify_idct(sym, [1.0, 0.5], H, W, L, C)
    l0 = y[:120].reshape(12, 10)
    want = np.zeros((12, 10))
    want[:8, :8], want[:8, 8:], want[8:, :8], want[8:, 8:] = 1, 2, 3, 4
    assert np.abs(l0 - want).max() < 1e-13
    assert np.abs(y[120:] - 4.0).max() < 1e-13 and y.size == 120 + 30
    sym[2] = 0
    sym[2, 4] = 16
    l0 = o.unpatchify_idct(sym, [1.0, 0.5], H, W, L, C)[:120].reshape(12, 10)
    pat = np.array([1, -1, -1, 1, 1, -1, -1, 1]) * 2.0
    assert np.abs(l0[8:, :8] - pat[None, :]).max() < 1e-13
    assert np.abs(l0[8:, 8:] - 4).max() < 1e-13 and np.abs(l0[:8, :8] - 1).max() < 1e-13


def pin_patchify_round_trip(o):
    """On planes whose sides are multiples of 8 the encoder's Patchify + DCT
    returns the integer coefficients the decoder started from, for every
    patch of a 2-channel pyramid."""
    H, W, L, C = 32, 64, 3, 2   # levels 32x64, 16x32, 8x16
    n = o.block_count(H, W, L, C)
    rng = np.random.Generator(np.random.PCG64(47))
    sym = rng.integers(-40, 41, (n, 64)).astype(np.int32)
    y = o.unpatchify_idct(sym, [1.0, 1.0, 1.0], H, W, L, C)
    assert np.abs(o.patchify_dct(y, H, W, L, C) - sym).max() < 1e-10
    # and the per-level step scales each level's latents exactly
    y2 = o.unpatchify_idct(sym, [1.0, 0.5, 0.25], H, W, L, C)
    off = 0
    for l, st in enumerate([1.0, 0.5, 0.25]):
        k = C * o.level_size(H, l) * o.level_size(W, l)
        assert np.abs(y2[off:off + k] - st * y[off:off + k]).max() < 1e-12
        off += k


def pin_decode_values_matches_decode(o):
    """Decoding real latents equal to the dequantised symbols is the integer
    decode (2 channels, 3 levels, ragged sizes)."""
    H, W, L, C = 11, 13, 3, 2
    dims = [L * C, 8, 3]
    rng = np.random.Generator(np.random.PCG64(53))
    q = rng.integers(-9, 10, o.latent_count(H, W, L, C)).astype(np.int32)
    steps = np.array([1.0, 0.5, 0.25])
    w = rng.normal(0.0, 0.3, o.param_count(dims))
    ref = o.decode(q, steps, w, H, W, L, C, dims, "relu", clamp=False)
    y = np.concatenate([o.dequant(q[a:b], steps[l]) for l, (a, b) in enumerate(
        _level_ranges(o, H, W, L, C))])
    assert np.array_equal(o.decode_values(y, w, H, W, L, C, dims, "relu", clamp=False), ref)


def _level_ranges(o, H, W, L, C):
    out, off = [], 0
    for l in range(L):
        k = C * o.level_size(H, l) * o.level_size(W, l)
        out.append((off, off + k))
        off += k
    return out


# --------------------------------------- modulation fusion (Sec. 3.1, App. A)
def pin_channel_stats_closed_form(o):
    """Population mean / std: (1, 2, 3, 4) -> 2.5, sqrt(5/4); (-1, 1, -1, 1)
    -> 0, 1 (dividing by N, not N - 1)."""
    mu, sd = o.channel_stats(np.array([[1.0, 2, 3, 4], [-1, 1, -1, 1]]))
    assert np.allclose(mu, [2.5, 0.0], atol=1e-15)
    assert np.allclose(sd, [np.sqrt(1.25), 1.0], atol=1e-15)


def pin_norm_modulate_moments(o):
    """Normalised features have mean 0 and population std 1 per channel;
    modulated ones have mean beta and std |gamma|."""
    rng = np.random.Generator(np.random.PCG64(61))
    f = rng.normal(3.0, 2.0, (5, 1000)) * rng.uniform(0.5, 4, (5, 1))
    mu, sd = o.channel_stats(f)
    z = o.norm_modulate(f, mu, sd, np.ones(5), np.zeros(5))
    assert np.abs(z.mean(axis=1)).max() < 1e-12 and np.abs(z.std(axis=1) - 1).max() < 1e-12
    g, b = rng.uniform(-2, 2, 5), rng.normal(0, 1, 5)
    z = o.norm_modulate(f, mu, sd, g, b)
    assert np.abs(z.mean(axis=1) - b).max() < 1e-12
    assert np.abs(z.std(axis=1) - np.abs(g)).max() < 1e-12


def pin_fusion_identity(o):
    """App. A: the linear layer on normalised, modulated features equals the
    fused layer (w', b') on the raw features, pixel by pixel; with
    gamma = sigma and beta = mu the fusion leaves (w, b) unchanged."""
    rng = np.random.Generator(np.random.PCG64(67))
    C, N, dout = 16, 300, 3
    f = rng.normal(1.0, 3.0, (C, N))
    w, b = rng.normal(0, 0.3, (dout, C)), rng.normal(0, 0.1, dout)
    g, be = rng.uniform(0.5, 1.5, C), rng.normal(0, 0.5, C)
    mu, sd = o.channel_stats(f)
    ref = w @ o.norm_modulate(f, mu, sd, g, be) + b[:, None]
    wf, bf = o.fuse_modulation(w, b, g, be, mu, sd)
    assert np.abs(wf @ f + bf[:, None] - ref).max() < 1e-12
    wi, bi = o.fuse_modulation(w, b, sd, mu, mu, sd)
    assert np.abs(wi - w).max() < 1e-15 and np.abs(bi - b).max() < 1e-15


def _fuse_last_layer(o, weights, dims, g, be, mu, sd):
    w = np.array(weights, dtype=np.float64)
    off = sum(dims[k + 1] * (dims[k] + 1) for k in range(len(dims) - 2))
    cf = dims[-2]
    wl = w[off:off + 3 * cf].reshape(3, cf)
    bl = w[off + 3 * cf: off + 3 * cf + 3]
    wf, bf = o.fuse_modulation(wl, bl, g, be, mu, sd)
    w[off:off + 3 * cf] = wf.ravel()
    w[off + 3 * cf: off + 3 * cf + 3] = bf
    return w


def pin_decode_modulated_equals_fused(o):
    """A whole decode: MLP^s -> normalise (the image's own mu, sigma) ->
    modulate -> MLP^i equals the plain decode with the fused last layer
    (unclamped, 2 channels, ragged sizes, both activations)."""
    H, W, L, C = 13, 17, 3, 2
    rng = np.random.Generator(np.random.PCG64(71))
    for act, dims in (("relu", [6, 12, 8, 3]), ("gelu", [6, 10, 3])):
        q = rng.integers(-9, 10, o.latent_count(H, W, L, C)).astype(np.int32)
        st = np.array([1.0, 0.5, 0.25])
        w = rng.normal(0, 0.4, o.param_count(dims))
        mu, sd = o.mlps_stats(q, st, w, H, W, L, C, dims, act)
        g, be = rng.uniform(0.5, 1.5, dims[-2]), rng.normal(0, 0.5, dims[-2])
        ref = o.decode_modulated(q, st, w, H, W, L, C, dims, act, g, be, mu, sd, clamp=False)
        got = o.decode(q, st, _fuse_last_layer(o, w, dims, g, be, mu, sd), H, W, L, C, dims, act,
                       clamp=False)
        assert np.abs(got - ref).max() < 1e-11 * max(1.0, np.abs(ref).max())


def pin_mlps_stats_bruteforce(o):
    """With MLP^s a single identity layer (W = I, b = 0, ReLU), its output is
    ReLU of the upsampled latents, whose per-channel moments numpy computes
    from the (pinned) upsampler directly."""
    H, W, L, C = 12, 20, 2, 1
    rng = np.random.Generator(np.random.PCG64(73))
    q = rng.integers(-7, 8, o.latent_count(H, W, L, C)).astype(np.int32)
    st = np.array([1.0, 0.5])
    dims = [2, 2, 3]
    w = np.concatenate([np.eye(2).ravel(), np.zeros(2), rng.normal(0, 1, 9)])
    mu, sd = o.mlps_stats(q, st, w, H, W, L, C, dims, "relu")
    l0 = q[:H * W].reshape(H, W) * 1.0
    l1 = o.upsample(q[H * W:].reshape(6, 10) * 0.5, H, W)
    f = np.maximum(np.stack([l0.ravel(), l1.ravel()]), 0.0)
    assert np.abs(mu - f.mean(axis=1)).max() < 1e-13
    assert np.abs(sd - f.std(axis=1)).max() < 1e-13


# --------------------------------------------------- Huffman coding (Sec. 3.3)
def _heap_huffman_cost(freq):
    """Cost (sum of weight x length) of an optimal prefix code, as the sum of
    the internal-node weights of Huffman's merge tree (heapq)."""
    import heapq
    h = [int(f) for f in freq if f > 0]
    heapq.heapify(h)
    cost = 0
    while len(h) > 1:
        a, b = heapq.heappop(h), heapq.heappop(h)
        cost += a + b
        heapq.heappush(h, a + b)
    return cost


def pin_huffman_textbook_example(o):
    """The classic six-symbol example (frequencies 45, 13, 12, 16, 9, 5 -- a:1
    b:3 c:3 d:3 e:4 f:4, cost 224)."""
    ln = o.huffman_lengths([45, 13, 12, 16, 9, 5], 15)
    assert ln.tolist() == [1, 3, 3, 3, 4, 4]
    assert int(np.dot(ln, [45, 13, 12, 16, 9, 5])) == 224


def pin_huffman_optimal_and_complete(o):
    """Without an effective length limit the lengths are optimal (cost of a
    heap-built Huffman tree) and complete (Kraft sum exactly 1); zero weights
    get no code; a single symbol gets length 1."""
    rng = np.random.Generator(np.random.PCG64(79))
    for n in (2, 3, 17, 200):
        f = rng.integers(1, 10 ** rng.integers(1, 6), n)
        f[rng.random(n) < 0.1] = 0
        if (f > 0).sum() < 2:
            f[:2] = [3, 5]
        ln = o.huffman_lengths(f, 24)
        assert int(np.dot(ln, f)) == _heap_huffman_cost(f)
        assert np.all((ln == 0) == (f == 0))
        assert sum(2.0 ** -l for l in ln if l > 0) == 1.0
    assert o.huffman_lengths([0, 7, 0], 5).tolist() == [0, 1, 0]


def pin_huffman_length_limited_optimal(o):
    """Fibonacci weights make an unlimited code 9 levels deep; with a limit of
    4 the lengths respect it, stay complete, and reach the least cost of all
    length vectors under the limit that satisfy Kraft's inequality (brute
    force over the non-increasing assignments, heavier symbols shorter)."""
    import itertools
    f = [1, 1, 2, 3, 5, 8, 13, 21, 34, 55]
    assert o.huffman_lengths(f, 24).max() == 9
    ln = o.huffman_lengths(f, 4)
    assert ln.max() <= 4 and sum(2.0 ** -l for l in ln) == 1.0
    best = None
    for combo in itertools.combinations_with_replacement(range(1, 5), len(f)):
        lens = sorted(combo, reverse=True)  # lightest symbol gets the longest code
        if sum(2.0 ** -l for l in lens) <= 1.0:
            c = sum(a * b for a, b in zip(f, lens))
            best = c if best is None or c < best else best
    assert int(np.dot(ln, f)) == best


def pin_huffman_hand_bits(o):
    """Lengths (1, 2, 2) give canonical codes 0, 10, 11: the stream
    (A, B, C, A) is the 6 bits 010110, MSB first: word 0x58000000."""
    tv, tl = o.huffman_table([7, -3, 12], [1, 2, 2])
    assert tv.tolist() == [7, -3, 12] and tl.tolist() == [1, 2, 2]
    w, nb = o.huffman_encode([7, -3, 12, 7], tv, tl)
    assert nb == 6 and w.tolist() == [0x58000000]
    assert o.huffman_decode(w, nb, tv, tl, 4).tolist() == [7, -3, 12, 7]
    # canonical order is (length, value): value 12 before 20 at equal length
    tv, tl = o.huffman_table([20, 5, 12], [2, 1, 2])
    assert tv.tolist() == [5, 12, 20] and tl.tolist() == [1, 2, 2]


def pin_huffman_round_trip(o):
    """ZpR-like streams (a few frequent values, a long tail) under a 12-bit
    limit decode back exactly; the bit count is sum(length); decoding past
    the end is refused."""
    rng = np.random.Generator(np.random.PCG64(83))
    syms = np.rint(rng.laplace(0, 3, 5000)).astype(np.int32)
    syms[rng.random(5000) < 0.1] = 300
    vals, counts = np.unique(syms, return_counts=True)
    ln = o.huffman_lengths(counts, 12)
    assert ln.max() <= 12
    tv, tl = o.huffman_table(vals, ln)
    w, nb = o.huffman_encode(syms, tv, tl)
    assert nb == int(np.dot(counts, ln))
    assert np.array_equal(o.huffman_decode(w, nb, tv, tl, syms.size), syms)
    try:
        o.huffman_decode(w, nb, tv, tl, syms.size + 1)
    except ValueError:
        pass
    else:
        raise AssertionError("decoding past the end was accepted")


PINS = [v for k, v in sorted(globals().items()) if k.startswith("pin_") and callable(v)]
