"""Seeded synthetic inputs shaped like PIC's decode workloads.

This module only draws random inputs and describes their shapes.  It holds
none of the decoder's arithmetic (no dequantisation, interpolation or MLP), so
both the fp64 oracle side and the CUDA side of the tests may use it.

Shapes follow the decoder's statement of the problem (Sec. 3.1, Eq. 1): an
H x W image is represented by L latent grids, level l (0 = full resolution)
of size ceil(H / 2^l) x ceil(W / 2^l) with C channels, and by the weights of
the synthesis MLP g_s (Sec. 4.1).  The paper evaluates on Kodak (24 images of
768 x 512) and on CLIC high-resolution images (Sec. 4.1 "Dataset"); neither
dataset is available, so seeded stand-ins are drawn instead:

* latent symbols: a discretised Laplacian, round(Laplace(0, scale)) clipped to
  +-clip, int32 -- the heavy-tailed, zero-peaked statistics of quantised
  transform-coded symbols (Sec. 3.2 quantises DCT coefficients of the latents);
* per-level quantisation step 2^-l;
* MLP weights W_k ~ N(0, 1/fan_in) in the nn.Linear layout [out][in], biases
  0.01 * N(0, 1); fp32, or fp16 (round-to-nearest-even of the draw) where the
  workload fixes fp16 weights.

Draw order for one image with generator PCG64(seed): for l = 0..L-1, for
c = 0..C-1 the level's symbols; then for k = 0..n-1 the weight matrix W_k
followed by the bias b_k.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

ACTS = ("relu", "gelu")
PRECISIONS = ("fp32", "fp16_tc")


def level_size(n: int, l: int) -> int:
    """ceil(n / 2^l): the side of pyramid level l for an image side n (Eq. 1)."""
    p = 1 << l
    return (n + p - 1) // p


def level_shapes(H: int, W: int, L: int):
    return [(level_size(H, l), level_size(W, l)) for l in range(L)]


def latent_count(H: int, W: int, L: int, C: int) -> int:
    return sum(C * h * w for h, w in level_shapes(H, W, L))


def param_count(dims) -> int:
    return sum(dims[k + 1] * dims[k] + dims[k + 1] for k in range(len(dims) - 1))


@dataclass(frozen=True)
class Workload:
    """One decode workload: image size, pyramid, MLP and input statistics."""

    name: str
    H: int
    W: int
    L: int
    C: int
    dims: tuple
    act: str
    weight_dtype: str          # "fp32" or "fp16": the dtype the weights are defined in
    lap_scale: float
    clip: int
    seeds: tuple               # one seed per image; len(seeds) = batch size
    precisions: tuple = ("fp32",)   # decoder paths that run this workload
    note: str = field(default="", compare=False)

    @property
    def B(self) -> int:
        return len(self.seeds)

    @property
    def pixels(self) -> int:
        return self.B * self.H * self.W

    @property
    def n_latents(self) -> int:
        return latent_count(self.H, self.W, self.L, self.C)

    @property
    def n_params(self) -> int:
        return param_count(self.dims)

    @property
    def macs_per_pixel(self) -> int:
        return sum(self.dims[k] * self.dims[k + 1] for k in range(len(self.dims) - 1))

    @property
    def hidden_per_pixel(self) -> int:
        return sum(self.dims[1:-1])

    def replace(self, **kw) -> "Workload":
        d = dict(self.__dict__)
        d.update(kw)
        return Workload(**d)


# The five decode workloads.  Kodak-sized images stand in for the Kodak set,
# 1080p and 2160p images for the CLIC high-resolution set.
WORKLOADS = {
    "c1": Workload("c1", H=256, W=256, L=4, C=1, dims=(4, 16, 16, 3), act="relu",
                   weight_dtype="fp32", lap_scale=2.0, clip=15, seeds=(0,),
                   note="256x256, 4 levels x 1 ch, 4-16-16-3 ReLU, fp32"),
    "c2": Workload("c2", H=512, W=768, L=7, C=1, dims=(7, 40, 40, 3), act="gelu",
                   weight_dtype="fp32", lap_scale=3.0, clip=31, seeds=(1,),
                   note="768x512 (Kodak size), 7 levels x 1 ch, 7-40-40-3 GELU, fp32"),
    "c3": Workload("c3", H=1080, W=1920, L=7, C=2, dims=(14, 64, 64, 3), act="relu",
                   weight_dtype="fp32", lap_scale=3.0, clip=31, seeds=(2,),
                   note="1920x1080, 7 levels x 2 ch, 14-64-64-3 ReLU, fp32"),
    "c4": Workload("c4", H=2160, W=3840, L=8, C=2, dims=(16, 64, 64, 64, 3), act="gelu",
                   weight_dtype="fp32", lap_scale=4.0, clip=63, seeds=(3,),
                   precisions=("fp32", "fp16_tc"),
                   note="3840x2160, 8 levels x 2 ch, 16-64-64-64-3 GELU, fp32 + fp16 copy"),
    "c5": Workload("c5", H=512, W=768, L=7, C=1, dims=(7, 64, 64, 3), act="relu",
                   weight_dtype="fp16", lap_scale=3.0, clip=31, seeds=tuple(range(100, 164)),
                   precisions=("fp16_tc",),
                   note="batch of 64 Kodak-sized images, 7-64-64-3 ReLU, fp16 weights"),
}

# The decoding-speed ablation over the synthesis network's width (Sec. 4.3,
# its decode-speed-versus-width experiment): the paper's own g_s -- L = 8
# single-channel latents, a 4-layer MLP with ReLU -- at widths 8, 16 (the
# paper's choice), 32 and 64, on batches of 64 Kodak-sized images.
for _w in (8, 16, 32, 64):
    WORKLOADS[f"w{_w}"] = Workload(
        f"w{_w}", H=512, W=768, L=8, C=1, dims=(8, _w, _w, _w, 3), act="relu",
        weight_dtype="fp16", lap_scale=3.0, clip=31, seeds=tuple(range(200, 264)),
        precisions=("fp32", "fp16_tc"),
        note=f"batch of 64 Kodak-sized images, 8 levels x 1 ch, 8-{_w}-{_w}-{_w}-3 ReLU, fp16 weights")
del _w


@dataclass
class Inputs:
    """Host arrays for a batch of B images of one workload."""

    wl: Workload
    latents: np.ndarray      # int32 [B, n_latents]: levels concatenated, each [C][H_l][W_l]
    steps: np.ndarray        # float32 [B, L]
    weights: np.ndarray      # float32 or float16 [B, n_params]: the defined weights
    weights_fp16: np.ndarray | None = None   # fp16 copy (RNE) of fp32 weights, for the TC path

    def weights_for(self, precision: str) -> np.ndarray:
        """The weight blob a decoder path consumes: fp32 for the CUDA-core path,
        fp16 for the tensor-core path."""
        if precision == "fp32":
            return self.weights.astype(np.float32)
        if self.weights.dtype == np.float16:
            return self.weights
        if self.weights_fp16 is None:
            self.weights_fp16 = self.weights.astype(np.float16)
        return self.weights_fp16

    def oracle_weights(self, precision: str) -> np.ndarray:
        """The weights the oracle uses as the definition: the defined weights
        (fp32 draw, or fp16 where the workload defines fp16 weights), exactly
        widened to fp64."""
        return self.weights.astype(np.float64)


def _draw_image(rng: np.random.Generator, H, W, L, C, dims, lap_scale, clip, weight_dtype):
    levels = []
    for l in range(L):
        h, w = level_size(H, l), level_size(W, l)
        for _c in range(C):
            q = np.clip(np.rint(rng.laplace(0.0, lap_scale, (h, w))), -clip, clip).astype(np.int32)
            levels.append(q.ravel())
    return np.concatenate(levels), _draw_weights(rng, dims, weight_dtype)


def _draw_weights(rng: np.random.Generator, dims, weight_dtype):
    params = []
    for k in range(len(dims) - 1):
        din, dout = dims[k], dims[k + 1]
        Wk = rng.standard_normal((dout, din)) / np.sqrt(din)
        bk = 0.01 * rng.standard_normal(dout)
        params.append(Wk.ravel())
        params.append(bk)
    p64 = np.concatenate(params)
    return p64.astype(np.float16) if weight_dtype == "fp16" else p64.astype(np.float32)


def make_inputs(wl: Workload | str, batch: int | None = None) -> Inputs:
    """Draws the inputs of a workload (all its images, or the first `batch`)."""
    if isinstance(wl, str):
        wl = WORKLOADS[wl]
    seeds = wl.seeds if batch is None else wl.seeds[:batch]
    lat, wts = [], []
    for s in seeds:
        rng = np.random.Generator(np.random.PCG64(s))
        q, w = _draw_image(rng, wl.H, wl.W, wl.L, wl.C, wl.dims, wl.lap_scale, wl.clip,
                           wl.weight_dtype)
        lat.append(q)
        wts.append(w)
    steps = np.array([[2.0 ** -l for l in range(wl.L)]] * len(seeds), dtype=np.float32)
    return Inputs(wl=wl, latents=np.stack(lat), steps=steps, weights=np.stack(wts))


def custom(name: str, H: int, W: int, L: int, C: int, dims, act: str = "relu",
           weight_dtype: str = "fp32", lap_scale: float = 3.0, clip: int = 31,
           seed: int = 0, batch: int = 1, precisions=("fp32",)) -> Workload:
    """A workload with arbitrary shapes (odd sizes, edge cases) for tests."""
    return Workload(name, H=H, W=W, L=L, C=C, dims=tuple(dims), act=act,
                    weight_dtype=weight_dtype, lap_scale=lap_scale, clip=clip,
                    seeds=tuple(seed + i for i in range(batch)), precisions=tuple(precisions))


def dct_blocks(n_blocks: int, seed: int, scale: float = 6.0, decay: float = 0.72,
               clip: int = 255) -> np.ndarray:
    """Synthetic quantised 8x8 DCT blocks, int32 [n][64] in raster order
    (row * 8 + col): coefficient (row, col) is round(Laplace(0, scale *
    decay^(row + col))) clipped to +-clip, so low frequencies are large and
    high frequencies mostly zero -- the statistics the entropy stage of the
    codec sees (Sec. 3.2 quantises DCT coefficients of the latents)."""
    rng = np.random.Generator(np.random.PCG64(seed))
    rc = np.add.outer(np.arange(8), np.arange(8)).ravel()
    scales = scale * decay ** rc
    q = np.rint(rng.laplace(0.0, 1.0, (n_blocks, 64)) * scales)
    return np.clip(q, -clip, clip).astype(np.int32)


def block_count(H: int, W: int, L: int, C: int) -> int:
    """Number of 8x8 patches of one pyramid, sum_l C ceil(H_l/8) ceil(W_l/8)
    (Sec. 3.2, Eq. 6: every latent plane is cut into 8x8 patches)."""
    return sum(C * ((h + 7) // 8) * ((w + 7) // 8) for h, w in level_shapes(H, W, L))


# Quantised DCT coefficients in place of integer latents (the input of the
# inverse DCT stage, Fig. 1).  Coefficient (u, v) of every patch is
# round(Laplace(0, DCT_GAIN * lap_scale * DCT_DECAY^(u+v))) clipped to
# +-DCT_CLIP: large at low frequencies, mostly zero at high ones, as in a
# JPEG-like coder.  DCT_GAIN = 4 gives decoded latents about the spread of
# the workload's integer latents (an orthonormal 8x8 transform keeps the
# energy: latent variance = sum_uv 2 (4 b 0.72^(u+v))^2 / 64 ~= 2.1 b^2,
# against 2 b^2 for Laplace(b) symbols).
DCT_GAIN = 4.0
DCT_DECAY = 0.72
DCT_CLIP = 255


@dataclass
class DctInputs:
    """Host arrays for B images whose latents arrive as DCT coefficients."""

    wl: Workload
    coeffs: np.ndarray       # int32 [B, n_blocks, 64], patch-major, raster within a patch
    steps: np.ndarray        # float32 [B, L]
    weights: np.ndarray      # as Inputs.weights

    def weights_for(self, precision: str) -> np.ndarray:
        if precision == "fp32" or self.weights.dtype == np.float16:
            return self.weights.astype(np.float32) if precision == "fp32" else self.weights
        return self.weights.astype(np.float16)


def make_dct_inputs(wl: Workload | str, batch: int | None = None) -> DctInputs:
    """Draws, per image, the DCT coefficients of every patch and then the MLP
    weights, from PCG64 seeded with (seed, 7) -- a stream apart from
    make_inputs' latents."""
    if isinstance(wl, str):
        wl = WORKLOADS[wl]
    seeds = wl.seeds if batch is None else wl.seeds[:batch]
    n = block_count(wl.H, wl.W, wl.L, wl.C)
    rc = np.add.outer(np.arange(8), np.arange(8)).ravel()
    scales = DCT_GAIN * wl.lap_scale * DCT_DECAY ** rc
    cs, ws = [], []
    for s in seeds:
        rng = np.random.Generator(np.random.PCG64([s, 7]))
        q = np.rint(rng.laplace(0.0, 1.0, (n, 64)) * scales)
        cs.append(np.clip(q, -DCT_CLIP, DCT_CLIP).astype(np.int32))
        ws.append(_draw_weights(rng, wl.dims, wl.weight_dtype))
    steps = np.array([[2.0 ** -l for l in range(wl.L)]] * len(seeds), dtype=np.float32)
    return DctInputs(wl=wl, coeffs=np.stack(cs), steps=steps, weights=np.stack(ws))


def zigzag_diagonals() -> np.ndarray:
    """Anti-diagonal u + v of each zigzag position 0..63: the diagonals of an
    8x8 block hold 1, 2, .., 8, 7, .., 1 positions, walked in turn."""
    return np.repeat(np.arange(15), [min(d + 1, 15 - d) for d in range(15)])


def zpr_streams(wl: Workload | str, batch: int | None = None, eob: int | None = None):
    """Seeded symbol streams in the ZpR format (Sec. 3.3, Fig. 2), one per
    image, for timing the inverse ZpR without an encoder: the coefficients of
    each patch are drawn directly in zigzag order -- position k with the
    Laplace scale of its frequency diagonal, as make_dct_inputs draws them --
    and written as the stream format reads: literals as themselves, every
    run of zeros before a literal as codes eob - 17 + n (n <= 16 zeros each),
    nothing after the last literal, then eob.  Returns (symbols int32 [total],
    per-image symbol counts int64 [B], n_blocks per image, eob)."""
    if isinstance(wl, str):
        wl = WORKLOADS[wl]
    eob = DCT_CLIP + 17 if eob is None else eob
    seeds = wl.seeds if batch is None else wl.seeds[:batch]
    n = block_count(wl.H, wl.W, wl.L, wl.C)
    scales = DCT_GAIN * wl.lap_scale * DCT_DECAY ** zigzag_diagonals()
    out, counts = [], []
    for s in seeds:
        rng = np.random.Generator(np.random.PCG64([s, 11]))
        z = np.clip(np.rint(rng.laplace(0.0, 1.0, (n, 64)) * scales), -DCT_CLIP, DCT_CLIP)
        z = z.astype(np.int32)
        blk, pos = np.nonzero(z)                          # literals, block-major, in position order
        first = np.r_[True, blk[1:] != blk[:-1]]
        prev = np.where(first, -1, np.r_[-1, pos[:-1]])
        run = pos - prev - 1                              # zeros before each literal
        ncode = (run + 15) // 16
        per_lit = ncode + 1                               # symbols each literal brings
        lits_per_blk = np.bincount(blk, minlength=n)
        sym_per_blk = np.bincount(blk, weights=per_lit, minlength=n).astype(np.int64) + 1
        blk_start = np.r_[0, np.cumsum(sym_per_blk)[:-1]]
        total = int(sym_per_blk.sum())
        stream = np.full(total, eob, dtype=np.int32)      # every slot not written below is a marker
        cum = np.cumsum(per_lit)                          # over all literals, block-major
        first_lit = np.r_[0, np.cumsum(lits_per_blk)[:-1]]
        lit_end = blk_start[blk] + cum - np.r_[0, cum][first_lit][blk]  # one past each literal
        stream[lit_end - 1] = z[blk, pos]                 # the literal, after its run codes
        # run codes: ncode slots before the literal, full runs of 16 then the remainder
        has = ncode > 0
        idx = np.repeat(np.nonzero(has)[0], ncode[has])
        j = np.arange(idx.size) - np.r_[0, np.cumsum(ncode[has])[:-1]].repeat(ncode[has])
        slot = lit_end[idx] - 1 - ncode[idx] + j
        left = run[idx] - 16 * j
        stream[slot] = eob - 17 + np.minimum(left, 16)
        out.append(stream)
        counts.append(total)
    return np.concatenate(out), np.array(counts, dtype=np.int64), n, eob


def make_modulation(B: int, cf: int, seed: int) -> np.ndarray:
    """Seeded stand-ins for g_m's modulation vectors and an image's feature
    statistics (g_m is a trained network, not available): float32 [B][4][cf]
    rows gamma ~ U(0.5, 1.5), beta ~ N(0, 0.5^2), mu ~ U(0, 2),
    sigma ~ U(0.3, 2)."""
    rng = np.random.Generator(np.random.PCG64([seed, 13]))
    m = np.empty((B, 4, cf))
    m[:, 0] = rng.uniform(0.5, 1.5, (B, cf))
    m[:, 1] = rng.normal(0.0, 0.5, (B, cf))
    m[:, 2] = rng.uniform(0.0, 2.0, (B, cf))
    m[:, 3] = rng.uniform(0.3, 2.0, (B, cf))
    return m.astype(np.float32)


HUFF_WORDS_PER_SUBSEQ = 8   # streams of a batch start on multiples of this many words


def huffman_code_lengths(counts: np.ndarray, p: int) -> np.ndarray:
    """Code lengths <= p for symbols with the given counts, for generating
    coded test inputs: Huffman's merge (heapq) for the depths, then lengths
    clamped to p and, while Kraft's sum exceeds 1, the longest code below p
    lengthened by one.  (A valid prefix code; the optimal one under the limit
    is the encoder's business.)"""
    import heapq
    n = len(counts)
    if n == 1:
        return np.array([1], dtype=np.int64)
    heap = [(int(c), i, [i]) for i, c in enumerate(counts)]
    heapq.heapify(heap)
    depth = np.zeros(n, dtype=np.int64)
    tick = n
    while len(heap) > 1:
        a, _, la = heapq.heappop(heap)
        b, _, lb = heapq.heappop(heap)
        depth[la + lb] += 1
        heapq.heappush(heap, (a + b, tick, la + lb))
        tick += 1
    ln = np.minimum(depth, p)
    order = np.argsort(-ln, kind="stable")
    while np.sum(2.0 ** -ln) > 1.0:
        j = next(i for i in order if ln[i] < p)
        ln[j] += 1
        order = np.argsort(-ln, kind="stable")
    return ln


def huffman_pack(symbols: np.ndarray, p: int):
    """One stream's image-specific canonical code and bits: returns
    (tab_value, tab_len) in canonical order (length, then value), the words
    (MSB first, padded to HUFF_WORDS_PER_SUBSEQ) and the number of bits."""
    vals, inv, counts = np.unique(symbols, return_inverse=True, return_counts=True)
    ln = huffman_code_lengths(counts, p)
    order = np.lexsort((vals, ln))                 # canonical: by length, then value
    code = np.zeros(len(vals), dtype=np.uint64)
    c = 0
    for k, i in enumerate(order):
        if k > 0:
            c = (c + 1) << int(ln[i] - ln[order[k - 1]])
        code[i] = c
    L = ln[inv].astype(np.uint64)
    pos = np.cumsum(L) - L
    n_bits = int(L.sum())
    n_words = -(-max(n_bits, 1) // 32)
    n_words = -(-n_words // HUFF_WORDS_PER_SUBSEQ) * HUFF_WORDS_PER_SUBSEQ
    words = np.zeros(n_words + 1, dtype=np.uint64)
    sh = np.uint64(64) - L - (pos & np.uint64(31))
    v = code[inv] << sh
    w = (pos >> np.uint64(5)).astype(np.int64)
    np.bitwise_or.at(words, w, v >> np.uint64(32))
    np.bitwise_or.at(words, w + 1, v & np.uint64(0xFFFFFFFF))
    return (vals[order].astype(np.int32), ln[order].astype(np.int32),
            words[:n_words].astype(np.uint32), n_bits)


def huffman_streams(wl: Workload | str, batch: int | None = None, p: int = 12):
    """The ZpR streams of zpr_streams, each Huffman-coded with its own
    table (Sec. 3.3): returns a dict with the concatenated words, word_off
    [B+1], n_bits [B], tab_value / tab_len [B][max_table] (zero-padded),
    sym_off [B+1], the symbols themselves and eob."""
    syms, counts, n_blk, eob = zpr_streams(wl, batch)
    starts = np.r_[0, np.cumsum(counts)]
    packs = [huffman_pack(syms[starts[b]:starts[b + 1]], p) for b in range(len(counts))]
    max_table = max(len(t[0]) for t in packs)
    B = len(packs)
    tv = np.zeros((B, max_table), np.int32)
    tl = np.zeros((B, max_table), np.int32)
    for b, (v, ln, _, _) in enumerate(packs):
        tv[b, :len(v)] = v
        tl[b, :len(ln)] = ln
    word_off = np.r_[0, np.cumsum([len(t[2]) for t in packs])].astype(np.int64)
    return {"words": np.concatenate([t[2] for t in packs]), "word_off": word_off,
            "n_bits": np.array([t[3] for t in packs], np.int64), "tab_value": tv,
            "tab_len": tl, "sym_off": starts.astype(np.int64), "symbols": syms,
            "n_blocks": n_blk, "eob": eob, "p": p}


def sample_pixels(H: int, W: int, n: int, seed: int) -> np.ndarray:
    """Flat pixel indices (y * W + x) to check at full size: the four corners,
    the middle of every border, and n seeded random positions."""
    rng = np.random.Generator(np.random.PCG64(seed))
    fixed = [(0, 0), (0, W - 1), (H - 1, 0), (H - 1, W - 1),
             (0, W // 2), (H - 1, W // 2), (H // 2, 0), (H // 2, W - 1)]
    ys = rng.integers(0, H, n)
    xs = rng.integers(0, W, n)
    idx = [y * W + x for y, x in fixed] + list(ys * W + xs)
    return np.unique(np.array(idx, dtype=np.int64))
