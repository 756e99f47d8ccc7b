"""Host-side checks of the seeded input generator (shapes, determinism,
statistics); no decoder arithmetic is involved."""
import numpy as np
import pytest

from paper_2609_09020_gb300 import workloads as wk


def test_level_shapes_match_ceiling_rule():
    assert wk.level_shapes(1080, 1920, 7)[-1] == (17, 30)
    assert wk.level_shapes(2160, 3840, 8)[-1] == (17, 30)
    assert wk.level_shapes(512, 768, 7)[-1] == (8, 12)


@pytest.mark.parametrize("name,lat,params", [
    ("c1", 87_040, 403), ("c2", 524_256, 2083), ("c3", 2 * 2_764_710, 5315),
    ("c4", 2 * 11_059_110, 9603), ("c5", 524_256, 4867)])
def test_workload_sizes(name, lat, params):
    wl = wk.WORKLOADS[name]
    assert wl.n_latents == lat
    assert wl.n_params == params


@pytest.mark.parametrize("name,recipe", [
    # image, levels x channels, MLP, activation, weight dtype, Laplace scale, clip, seeds
    ("c1", (256, 256, 4, 1, (4, 16, 16, 3), "relu", "fp32", 2.0, 15, (0,))),
    ("c2", (512, 768, 7, 1, (7, 40, 40, 3), "gelu", "fp32", 3.0, 31, (1,))),
    ("c3", (1080, 1920, 7, 2, (14, 64, 64, 3), "relu", "fp32", 3.0, 31, (2,))),
    ("c4", (2160, 3840, 8, 2, (16, 64, 64, 64, 3), "gelu", "fp32", 4.0, 63, (3,))),
    ("c5", (512, 768, 7, 1, (7, 64, 64, 3), "relu", "fp16", 3.0, 31, tuple(range(100, 164)))),
])
def test_workload_recipes(name, recipe):
    wl = wk.WORKLOADS[name]
    assert (wl.H, wl.W, wl.L, wl.C, wl.dims, wl.act, wl.weight_dtype, wl.lap_scale, wl.clip,
            wl.seeds) == recipe


def test_width_sweep_is_the_papers_net_at_four_widths():
    for w in (8, 16, 32, 64):
        wl = wk.WORKLOADS[f"w{w}"]
        assert (wl.H, wl.W, wl.L, wl.C, wl.act, wl.B) == (512, 768, 8, 1, "relu", 64)
        assert wl.dims == (8, w, w, w, 3)


def test_generator_is_deterministic_and_bounded():
    a = wk.make_inputs("c1")
    b = wk.make_inputs("c1")
    assert np.array_equal(a.latents, b.latents) and np.array_equal(a.weights, b.weights)
    assert a.latents.dtype == np.int32 and a.latents.shape == (1, 87_040)
    assert np.abs(a.latents).max() <= 15
    assert a.steps.tolist() == [[1.0, 0.5, 0.25, 0.125]]
    # discretised Laplace(0, 2): P(q = 0) = 1 - exp(-1/4) ~ 0.221
    p0 = np.mean(a.latents == 0)
    assert 0.20 < p0 < 0.24


def test_batch_uses_one_seed_per_image():
    x = wk.make_inputs("c5", batch=3)
    assert x.latents.shape == (3, 524_256) and x.weights.dtype == np.float16
    assert not np.array_equal(x.latents[0], x.latents[1])
    y = wk.make_inputs(wk.WORKLOADS["c5"].replace(seeds=(101,)))
    assert np.array_equal(y.latents[0], x.latents[1])


def test_fp16_copy_is_round_to_nearest():
    x = wk.make_inputs(wk.custom("t", 8, 8, 2, 1, (2, 4, 3)))
    h = x.weights_for("fp16_tc")
    assert h.dtype == np.float16
    assert np.array_equal(h, x.weights.astype(np.float16))


def test_sample_pixels_include_corners():
    p = wk.sample_pixels(10, 7, 20, 0)
    for idx in (0, 6, 63, 69):
        assert idx in p
    assert p.min() >= 0 and p.max() < 70


def test_zpr_streams_are_the_oracle_encoding(orc):
    """The direct stream generator writes exactly what the oracle's ZpR
    encoder makes of the same coefficients (redrawn here in zigzag order and
    scattered to raster order with the oracle's zigzag table)."""
    wl = wk.custom("z", H=40, W=72, L=3, C=2, dims=(6, 8, 3), batch=3, lap_scale=3.0)
    s, counts, n, eob = wk.zpr_streams(wl)
    assert n == orc.block_count(40, 72, 3, 2) and eob == wk.DCT_CLIP + 17
    assert counts.sum() == s.size
    order = orc.zigzag()
    scales = wk.DCT_GAIN * wl.lap_scale * wk.DCT_DECAY ** wk.zigzag_diagonals()
    off = 0
    for b in range(3):
        rng = np.random.Generator(np.random.PCG64([wl.seeds[b], 11]))
        z = np.clip(np.rint(rng.laplace(0.0, 1.0, (n, 64)) * scales), -255, 255).astype(np.int32)
        raster = np.zeros_like(z)
        raster[:, order] = z
        assert np.array_equal(orc.zpr_encode(raster, eob), s[off:off + counts[b]])
        off += counts[b]


def test_zigzag_diagonals(orc):
    order = orc.zigzag()
    assert np.array_equal(wk.zigzag_diagonals(), order // 8 + order % 8)


def test_huffman_pack_is_the_oracle_encoding(orc):
    """The stream generator's table is a valid canonical code under the
    precision (Kraft <= 1, canonical order) and its bits are exactly the
    oracle's encoding with that table; the oracle decodes them back."""
    rng = np.random.Generator(np.random.PCG64(89))
    for p, syms in ((12, np.rint(rng.laplace(0, 4, 3000)).astype(np.int32)),
                    (5, rng.integers(-3, 4, 500).astype(np.int32)),
                    (4, np.full(37, 9, np.int32))):
        tv, tl, words, nb = wk.huffman_pack(syms, p)
        assert tl.max() <= p and np.sum(2.0 ** -tl.astype(float)) <= 1.0
        ctv, ctl = orc.huffman_table(tv, tl)
        assert np.array_equal(ctv, tv) and np.array_equal(ctl, tl)
        w, nb2 = orc.huffman_encode(syms, tv, tl)
        assert nb2 == nb and np.array_equal(words[:len(w)], w) and not words[len(w):].any()
        assert len(words) % wk.HUFF_WORDS_PER_SUBSEQ == 0
        assert np.array_equal(orc.huffman_decode(words, nb, tv, tl, syms.size), syms)
