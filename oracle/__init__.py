"""fp64 CPU oracle of the PIC decode synthesis (Sec. 3.1 Eq. 1, Sec. 4.1, App. A).

TEST INFRASTRUCTURE ONLY: the parity oracle for the CUDA decoder.  Only the
tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py``
import this module.  It shares no code with the CUDA path and never imports
the ``paper_2609_09020_gb300`` package.

The arithmetic lives in ``pic_oracle.c`` (plain C, double precision, compiled
with ``-O2 -ffp-contract=off``); this module compiles it with gcc and marshals
numpy arrays through ctypes.

Parity status of each function (what pins it is in tests/test_oracle.py):
  dequant             pinned (exact integer x power-of-two products)
  bilinear/upsample   pinned (constants, affine grids, brute-force
                      half-pixel interpolation, hand-computed grids)
  mlp                 pinned (zero/identity weights, hand-computed layers,
                      GELU closed forms)
  decode              pinned (hand-computed 4x4 image, reductions to the
                      pieces above, planted-mistake runs)
  decode_values       pinned (equals decode on dequantised symbols)
  dct8x8 / idct8x8    pinned (scipy's orthonormal DCT-II/III, DC-only and
                      one-dimensional closed forms, Parseval, inverse pair)
  patchify/unpatchify pinned (hand-placed DC patches on ragged planes,
                      block counts of the decode workloads, round trip)
  zigzag / ZpR / iZpR pinned (hand-worked stream, JPEG zigzag table start,
                      round trips, malformed streams)
  Huffman code        pinned (textbook example lengths, Kraft equality,
                      optimal cost against a heap-built Huffman tree,
                      length limit, hand-worked bits, round trips)
  modulation fusion   pinned (closed-form statistics, normalised moments,
                      fused == un-fused on random data and on whole decodes,
                      the identity special case, brute-force statistics)
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "pic_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "libpic_oracle.so")

ACT_RELU = 0
ACT_GELU = 1
ACTS = {"relu": ACT_RELU, "gelu": ACT_GELU}

_lock = threading.Lock()
_lib = None


def compile_oracle(src: str = _SRC, out: str = _LIB_PATH, extra_flags=()) -> str:
    """Compiles the oracle C file into a shared library with gcc; returns its path."""
    os.makedirs(os.path.dirname(out), exist_ok=True)
    cmd = ["gcc", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fopenmp", "-shared",
           "-fPIC", "-std=c11", *extra_flags, "-o", out + ".tmp", src, "-lm"]
    subprocess.run(cmd, check=True, capture_output=True, text=True)
    os.replace(out + ".tmp", out)
    return out


def _needs_build() -> bool:
    return (not os.path.exists(_LIB_PATH)) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC)


def _declare(lib):
    c_int, c_i64, c_dbl = ctypes.c_int, ctypes.c_int64, ctypes.c_double
    p = ctypes.c_void_p
    lib.pic_oracle_level_size.argtypes = [c_int, c_int]
    lib.pic_oracle_level_size.restype = c_int
    lib.pic_oracle_latent_count.argtypes = [c_int, c_int, c_int, c_int]
    lib.pic_oracle_latent_count.restype = c_i64
    lib.pic_oracle_param_count.argtypes = [c_int, p]
    lib.pic_oracle_param_count.restype = c_i64
    lib.pic_oracle_dequant.argtypes = [p, c_i64, c_dbl, p]
    lib.pic_oracle_dequant.restype = None
    lib.pic_oracle_bilinear_at.argtypes = [p, c_int, c_int, c_int, c_int, c_int, c_int]
    lib.pic_oracle_bilinear_at.restype = c_dbl
    lib.pic_oracle_upsample.argtypes = [p, c_int, c_int, c_int, c_int, p]
    lib.pic_oracle_upsample.restype = None
    lib.pic_oracle_act.argtypes = [c_dbl, c_int]
    lib.pic_oracle_act.restype = c_dbl
    lib.pic_oracle_mlp.argtypes = [p, p, c_int, p, c_int, p]
    lib.pic_oracle_mlp.restype = c_int
    lib.pic_oracle_clamp01.argtypes = [c_dbl]
    lib.pic_oracle_clamp01.restype = c_dbl
    lib.pic_oracle_to_u8.argtypes = [c_dbl]
    lib.pic_oracle_to_u8.restype = c_int
    lib.pic_oracle_decode.argtypes = [p, p, p, c_int, c_int, c_int, p, c_int, c_int,
                                      c_int, c_int, p, p, c_int]
    lib.pic_oracle_decode.restype = c_int
    lib.pic_oracle_decode_pixels.argtypes = [p, p, p, c_int, c_int, c_int, p, c_int, c_int,
                                             c_int, c_int, p, c_i64, p, p]
    lib.pic_oracle_decode_pixels.restype = c_int
    lib.pic_oracle_zigzag.argtypes = [p]
    lib.pic_oracle_zigzag.restype = None
    lib.pic_oracle_zpr_encode.argtypes = [p, c_i64, ctypes.c_int32, p, c_i64]
    lib.pic_oracle_zpr_encode.restype = c_i64
    lib.pic_oracle_izpr.argtypes = [p, c_i64, ctypes.c_int32, p, c_i64]
    lib.pic_oracle_izpr.restype = c_int
    lib.pic_oracle_decode_values.argtypes = [p, p, c_int, c_int, c_int, p, c_int, c_int, c_int,
                                             c_int, p, c_int]
    lib.pic_oracle_decode_values.restype = c_int
    lib.pic_oracle_dct8x8.argtypes = [p, p]
    lib.pic_oracle_dct8x8.restype = None
    lib.pic_oracle_idct8x8.argtypes = [p, p]
    lib.pic_oracle_idct8x8.restype = None
    lib.pic_oracle_block_count.argtypes = [c_int, c_int, c_int, c_int]
    lib.pic_oracle_block_count.restype = c_i64
    lib.pic_oracle_patchify_dct.argtypes = [p, c_int, c_int, c_int, c_int, p]
    lib.pic_oracle_patchify_dct.restype = c_int
    lib.pic_oracle_unpatchify_idct.argtypes = [p, p, c_int, c_int, c_int, c_int, p]
    lib.pic_oracle_unpatchify_idct.restype = c_int
    lib.pic_oracle_channel_stats.argtypes = [p, c_int, c_i64, p, p]
    lib.pic_oracle_channel_stats.restype = None
    lib.pic_oracle_norm_modulate.argtypes = [p, c_int, c_i64, p, p, p, p, p]
    lib.pic_oracle_norm_modulate.restype = None
    lib.pic_oracle_fuse_modulation.argtypes = [p, p, c_int, c_int, p, p, p, p, p, p]
    lib.pic_oracle_fuse_modulation.restype = None
    lib.pic_oracle_mlps_stats.argtypes = [p, p, p, c_int, c_int, c_int, p, c_int, c_int, c_int,
                                          p, p, p]
    lib.pic_oracle_mlps_stats.restype = c_int
    lib.pic_oracle_decode_modulated.argtypes = [p, p, p, c_int, c_int, c_int, p, c_int, c_int,
                                                p, p, p, p, c_int, c_int, p, p, c_int]
    lib.pic_oracle_decode_modulated.restype = c_int
    lib.pic_oracle_huffman_lengths.argtypes = [p, c_int, c_int, p]
    lib.pic_oracle_huffman_lengths.restype = c_int
    lib.pic_oracle_huffman_table.argtypes = [p, p, c_int, p, p]
    lib.pic_oracle_huffman_table.restype = c_int
    lib.pic_oracle_huffman_encode.argtypes = [p, c_i64, p, p, c_int, p, c_i64]
    lib.pic_oracle_huffman_encode.restype = c_i64
    lib.pic_oracle_huffman_decode.argtypes = [p, c_i64, p, p, c_int, p, c_i64]
    lib.pic_oracle_huffman_decode.restype = c_int
    return lib


def load(path: str | None = None):
    """Returns the ctypes handle of the oracle library, compiling it if needed.

    With ``path`` given, loads that (already compiled) library instead; the
    planted-mistake tests use this for mutated copies of the oracle."""
    global _lib
    if path is not None:
        return Oracle(_declare(ctypes.CDLL(path)))
    with _lock:
        if _lib is None:
            if _needs_build():
                compile_oracle()
            _lib = Oracle(_declare(ctypes.CDLL(_LIB_PATH)))
    return _lib


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


class Oracle:
    """numpy front end of one compiled copy of the oracle library."""

    def __init__(self, lib):
        self.lib = lib

    # ---- shapes -------------------------------------------------------
    def level_size(self, n: int, l: int) -> int:
        return int(self.lib.pic_oracle_level_size(n, l))

    def latent_count(self, H: int, W: int, L: int, C: int) -> int:
        return int(self.lib.pic_oracle_latent_count(H, W, L, C))

    def param_count(self, dims) -> int:
        d = np.ascontiguousarray(dims, dtype=np.int32)
        return int(self.lib.pic_oracle_param_count(len(d) - 1, _ptr(d)))

    # ---- pieces ------------------------------------------------------
    def dequant(self, q: np.ndarray, step: float) -> np.ndarray:
        q = np.ascontiguousarray(q, dtype=np.int32)
        y = np.empty(q.shape, dtype=np.float64)
        self.lib.pic_oracle_dequant(_ptr(q), q.size, float(step), _ptr(y))
        return y

    def bilinear_at(self, g: np.ndarray, H: int, W: int, x: int, y: int) -> float:
        g = np.ascontiguousarray(g, dtype=np.float64)
        return float(self.lib.pic_oracle_bilinear_at(_ptr(g), g.shape[0], g.shape[1], H, W, x, y))

    def upsample(self, g: np.ndarray, H: int, W: int) -> np.ndarray:
        g = np.ascontiguousarray(g, dtype=np.float64)
        out = np.empty((H, W), dtype=np.float64)
        self.lib.pic_oracle_upsample(_ptr(g), g.shape[0], g.shape[1], H, W, _ptr(out))
        return out

    def act(self, z: float, act: str) -> float:
        return float(self.lib.pic_oracle_act(float(z), ACTS[act]))

    def mlp(self, feat: np.ndarray, weights: np.ndarray, dims, act: str) -> np.ndarray:
        feat = np.ascontiguousarray(feat, dtype=np.float64)
        w = np.ascontiguousarray(weights, dtype=np.float64)
        d = np.ascontiguousarray(dims, dtype=np.int32)
        out = np.empty(int(d[-1]), dtype=np.float64)
        rc = self.lib.pic_oracle_mlp(_ptr(feat), _ptr(w), len(d) - 1, _ptr(d), ACTS[act], _ptr(out))
        if rc != 0:
            raise ValueError("oracle mlp rejected the dims")
        return out

    def clamp01(self, v: float) -> float:
        return float(self.lib.pic_oracle_clamp01(float(v)))

    def to_u8(self, v: float) -> int:
        return int(self.lib.pic_oracle_to_u8(float(v)))

    # ---- whole decode --------------------------------------------------
    def decode(self, latents, steps, weights, H, W, L, C, dims, act, clamp=True,
               nthreads: int = 1) -> np.ndarray:
        """Decodes one image; returns planar fp64 [3][H][W]."""
        q = np.ascontiguousarray(latents, dtype=np.int32).ravel()
        s = np.ascontiguousarray(steps, dtype=np.float64).ravel()
        w = np.ascontiguousarray(weights, dtype=np.float64).ravel()
        d = np.ascontiguousarray(dims, dtype=np.int32)
        if q.size != self.latent_count(H, W, L, C) or s.size != L or w.size != self.param_count(d):
            raise ValueError("oracle decode: buffer sizes do not match the shapes")
        out = np.empty((3, H, W), dtype=np.float64)
        work = np.empty(max(q.size, 1), dtype=np.float64)
        rc = self.lib.pic_oracle_decode(_ptr(q), _ptr(s), _ptr(w), L, C, len(d) - 1, _ptr(d),
                                        ACTS[act], int(bool(clamp)), H, W, _ptr(out), _ptr(work),
                                        int(nthreads))
        if rc != 0:
            raise ValueError("oracle decode rejected the arguments")
        return out

    def decode_pixels(self, latents, steps, weights, H, W, L, C, dims, act, pix,
                      clamp=True) -> np.ndarray:
        """Decodes the pixels with flat indices ``pix`` (y * W + x); returns [n][3]."""
        q = np.ascontiguousarray(latents, dtype=np.int32).ravel()
        s = np.ascontiguousarray(steps, dtype=np.float64).ravel()
        w = np.ascontiguousarray(weights, dtype=np.float64).ravel()
        d = np.ascontiguousarray(dims, dtype=np.int32)
        p = np.ascontiguousarray(pix, dtype=np.int64).ravel()
        if q.size != self.latent_count(H, W, L, C) or s.size != L or w.size != self.param_count(d):
            raise ValueError("oracle decode_pixels: buffer sizes do not match the shapes")
        out = np.empty((p.size, 3), dtype=np.float64)
        work = np.empty(max(q.size, 1), dtype=np.float64)
        rc = self.lib.pic_oracle_decode_pixels(_ptr(q), _ptr(s), _ptr(w), L, C, len(d) - 1,
                                               _ptr(d), ACTS[act], int(bool(clamp)), H, W,
                                               _ptr(p), p.size, _ptr(out), _ptr(work))
        if rc != 0:
            raise ValueError("oracle decode_pixels rejected the arguments")
        return out

    def decode_values(self, latents, weights, H, W, L, C, dims, act, clamp=True,
                      nthreads: int = 1) -> np.ndarray:
        """Decodes one image from real-valued latents (the iDCT output);
        returns planar fp64 [3][H][W]."""
        y = np.ascontiguousarray(latents, dtype=np.float64).ravel()
        w = np.ascontiguousarray(weights, dtype=np.float64).ravel()
        d = np.ascontiguousarray(dims, dtype=np.int32)
        if y.size != self.latent_count(H, W, L, C) or w.size != self.param_count(d):
            raise ValueError("oracle decode_values: buffer sizes do not match the shapes")
        out = np.empty((3, H, W), dtype=np.float64)
        rc = self.lib.pic_oracle_decode_values(_ptr(y), _ptr(w), L, C, len(d) - 1, _ptr(d),
                                               ACTS[act], int(bool(clamp)), H, W, _ptr(out),
                                               int(nthreads))
        if rc != 0:
            raise ValueError("oracle decode_values rejected the arguments")
        return out

    # ---- Patchify / DCT and their inverses (Sec. 3.2, Eqs. 5-7) --------
    def dct8x8(self, x: np.ndarray) -> np.ndarray:
        x = np.ascontiguousarray(x, dtype=np.float64).reshape(8, 8)
        S = np.empty((8, 8), dtype=np.float64)
        self.lib.pic_oracle_dct8x8(_ptr(x), _ptr(S))
        return S

    def idct8x8(self, S: np.ndarray) -> np.ndarray:
        S = np.ascontiguousarray(S, dtype=np.float64).reshape(8, 8)
        x = np.empty((8, 8), dtype=np.float64)
        self.lib.pic_oracle_idct8x8(_ptr(S), _ptr(x))
        return x

    def block_count(self, H: int, W: int, L: int, C: int) -> int:
        return int(self.lib.pic_oracle_block_count(H, W, L, C))

    def patchify_dct(self, latents, H, W, L, C) -> np.ndarray:
        """Encoder side: real latents (pyramid layout) -> DCT coefficients [n][64]."""
        y = np.ascontiguousarray(latents, dtype=np.float64).ravel()
        if y.size != self.latent_count(H, W, L, C):
            raise ValueError("patchify_dct: latent count does not match the shapes")
        out = np.empty((self.block_count(H, W, L, C), 64), dtype=np.float64)
        if self.lib.pic_oracle_patchify_dct(_ptr(y), H, W, L, C, _ptr(out)) != 0:
            raise ValueError("patchify_dct rejected the shapes")
        return out

    def unpatchify_idct(self, symbols, steps, H, W, L, C) -> np.ndarray:
        """Decoder side: int coefficients [n][64] x per-level step -> iDCT ->
        real latents in the pyramid layout (fp64)."""
        s = np.ascontiguousarray(symbols, dtype=np.int32).ravel()
        st = np.ascontiguousarray(steps, dtype=np.float64).ravel()
        if s.size != 64 * self.block_count(H, W, L, C) or st.size != L:
            raise ValueError("unpatchify_idct: buffer sizes do not match the shapes")
        out = np.empty(self.latent_count(H, W, L, C), dtype=np.float64)
        if self.lib.pic_oracle_unpatchify_idct(_ptr(s), _ptr(st), H, W, L, C, _ptr(out)) != 0:
            raise ValueError("unpatchify_idct rejected the shapes")
        return out

    # ---- modulation fusion (Sec. 3.1 Eqs. 2-3, App. A) -----------------
    def channel_stats(self, f):
        """Population mean and std per channel of f [C][N]."""
        f = np.ascontiguousarray(f, dtype=np.float64)
        C, N = f.shape
        mu, sd = np.empty(C), np.empty(C)
        self.lib.pic_oracle_channel_stats(_ptr(f), C, N, _ptr(mu), _ptr(sd))
        return mu, sd

    def norm_modulate(self, f, mu, sigma, gamma, beta):
        f = np.ascontiguousarray(f, dtype=np.float64)
        C, N = f.shape
        a = [np.ascontiguousarray(v, dtype=np.float64) for v in (mu, sigma, gamma, beta)]
        out = np.empty_like(f)
        self.lib.pic_oracle_norm_modulate(_ptr(f), C, N, *[_ptr(v) for v in a], _ptr(out))
        return out

    def fuse_modulation(self, w, b, gamma, beta, mu, sigma):
        """App. A: (w', b') of the fused MLP^i layer; w [dout][C]."""
        w = np.ascontiguousarray(w, dtype=np.float64)
        dout, C = w.shape
        a = [np.ascontiguousarray(v, dtype=np.float64) for v in (b, gamma, beta, mu, sigma)]
        wo, bo = np.empty_like(w), np.empty(dout)
        self.lib.pic_oracle_fuse_modulation(_ptr(w), _ptr(a[0]), dout, C, *[_ptr(v) for v in a[1:]],
                                            _ptr(wo), _ptr(bo))
        return wo, bo

    def mlps_stats(self, latents, steps, weights, H, W, L, C, dims, act):
        """mu, sigma of the MLP^s output of one image over its pixels."""
        q = np.ascontiguousarray(latents, dtype=np.int32).ravel()
        s = np.ascontiguousarray(steps, dtype=np.float64).ravel()
        w = np.ascontiguousarray(weights, dtype=np.float64).ravel()
        d = np.ascontiguousarray(dims, dtype=np.int32)
        cf = int(d[-2])
        mu, sd = np.empty(cf), np.empty(cf)
        work = np.empty(max(q.size, 1))
        rc = self.lib.pic_oracle_mlps_stats(_ptr(q), _ptr(s), _ptr(w), L, C, len(d) - 1, _ptr(d),
                                            ACTS[act], H, W, _ptr(mu), _ptr(sd), _ptr(work))
        if rc != 0:
            raise ValueError("mlps_stats rejected the arguments")
        return mu, sd

    def decode_modulated(self, latents, steps, weights, H, W, L, C, dims, act, gamma, beta, mu,
                         sigma, clamp=True, nthreads: int = 1):
        """Un-fused decode: MLP^s, normalise, modulate, MLP^i, clamp -> [3][H][W]."""
        q = np.ascontiguousarray(latents, dtype=np.int32).ravel()
        s = np.ascontiguousarray(steps, dtype=np.float64).ravel()
        w = np.ascontiguousarray(weights, dtype=np.float64).ravel()
        d = np.ascontiguousarray(dims, dtype=np.int32)
        a = [np.ascontiguousarray(v, dtype=np.float64) for v in (gamma, beta, mu, sigma)]
        if q.size != self.latent_count(H, W, L, C) or w.size != self.param_count(d):
            raise ValueError("decode_modulated: buffer sizes do not match the shapes")
        out = np.empty((3, H, W))
        work = np.empty(max(q.size, 1))
        rc = self.lib.pic_oracle_decode_modulated(_ptr(q), _ptr(s), _ptr(w), L, C, len(d) - 1,
                                                  _ptr(d), ACTS[act], int(bool(clamp)),
                                                  *[_ptr(v) for v in a], H, W, _ptr(out),
                                                  _ptr(work), int(nthreads))
        if rc != 0:
            raise ValueError("decode_modulated rejected the arguments")
        return out

    # ---- Huffman coding (Sec. 3.3) -------------------------------------
    def huffman_lengths(self, freq, max_len: int) -> np.ndarray:
        f = np.ascontiguousarray(freq, dtype=np.int64)
        out = np.empty(f.size, dtype=np.int32)
        if self.lib.pic_oracle_huffman_lengths(_ptr(f), f.size, int(max_len), _ptr(out)) != 0:
            raise ValueError("huffman_lengths: no code under that length limit")
        return out

    def huffman_table(self, values, lengths):
        """(values, lengths) of the coded symbols in canonical order."""
        v = np.ascontiguousarray(values, dtype=np.int32)
        ln = np.ascontiguousarray(lengths, dtype=np.int32)
        tv, tl = np.empty(v.size, np.int32), np.empty(v.size, np.int32)
        m = self.lib.pic_oracle_huffman_table(_ptr(v), _ptr(ln), v.size, _ptr(tv), _ptr(tl))
        if m < 0:
            raise ValueError("huffman_table rejected the arguments")
        return tv[:m].copy(), tl[:m].copy()

    def huffman_encode(self, syms, tab_value, tab_len):
        """-> (uint32 words, number of bits)."""
        s = np.ascontiguousarray(syms, dtype=np.int32)
        tv = np.ascontiguousarray(tab_value, dtype=np.int32)
        tl = np.ascontiguousarray(tab_len, dtype=np.int32)
        cap = (s.size * int(tl.max(initial=1)) + 31) // 32 + 1
        words = np.empty(cap, dtype=np.uint32)
        nb = self.lib.pic_oracle_huffman_encode(_ptr(s), s.size, _ptr(tv), _ptr(tl), tv.size,
                                                _ptr(words), cap)
        if nb < 0:
            raise ValueError("huffman_encode: symbol not in the table")
        return words[:(nb + 31) // 32].copy(), int(nb)

    def huffman_decode(self, words, n_bits, tab_value, tab_len, n_out):
        w = np.ascontiguousarray(words, dtype=np.uint32)
        tv = np.ascontiguousarray(tab_value, dtype=np.int32)
        tl = np.ascontiguousarray(tab_len, dtype=np.int32)
        out = np.empty(n_out, dtype=np.int32)
        if self.lib.pic_oracle_huffman_decode(_ptr(w), int(n_bits), _ptr(tv), _ptr(tl), tv.size,
                                              _ptr(out), int(n_out)) != 0:
            raise ValueError("huffman_decode: malformed bit stream")
        return out

    # ---- ZpR / inverse ZpR (Sec. 3.3, Algorithm 1) ---------------------
    def zigzag(self) -> np.ndarray:
        order = np.empty(64, dtype=np.int32)
        self.lib.pic_oracle_zigzag(_ptr(order))
        return order

    def zpr_encode(self, coeffs: np.ndarray, eob: int) -> np.ndarray:
        """Forward ZpR of blocks [n][64] (raster order) -> int32 symbol stream."""
        c = np.ascontiguousarray(coeffs, dtype=np.int32).reshape(-1, 64)
        cap = c.shape[0] * 66 + 16
        out = np.empty(cap, dtype=np.int32)
        n = self.lib.pic_oracle_zpr_encode(_ptr(c), c.shape[0], int(eob), _ptr(out), cap)
        if n < 0:
            raise ValueError("zpr_encode: literal collides with the run codes, or overflow")
        return out[:n].copy()

    def izpr(self, symbols: np.ndarray, eob: int, n_blocks: int) -> np.ndarray:
        """Inverse ZpR -> int32 blocks [n_blocks][64] in raster order."""
        s = np.ascontiguousarray(symbols, dtype=np.int32)
        out = np.empty((n_blocks, 64), dtype=np.int32)
        rc = self.lib.pic_oracle_izpr(_ptr(s), s.size, int(eob), _ptr(out), n_blocks)
        if rc != 0:
            raise ValueError("izpr: malformed symbol stream")
        return out


def build() -> str:
    """Compiles the oracle library (used by the build step); returns its path."""
    with _lock:
        return compile_oracle()
