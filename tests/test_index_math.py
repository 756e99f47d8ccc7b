"""Index and transform arithmetic of the upstream kernels, restated and checked on
the CPU (no GPU): the inverse DCT's division by invariant integers and its
8-point butterfly, the inverse ZpR's segmented-scan operator and the bound
on the Huffman final decode's packed row offsets.

Patch -> (image, plane row) uses division by invariant integers (Granlund &
Montgomery 1994): for 32-bit n and d, floor(n / d) = the high 64 bits of
n * inv with inv = ceil(2^64 / d), computed on the host as (2^64 - 1) // d + 1
(d == 1 stored as inv == 0, meaning n itself).  With inv d = 2^64 + e,
0 <= e < d, the product over 2^64 is n / d + n e / (d 2^64), and the error
term is below 2^-32 <= 1/d, so it never crosses the next integer.
"""
import os
import re

import numpy as np

M64 = (1 << 64) - 1


def udiv_inv(d):
    return M64 // d + 1 if d > 1 else 0


def udiv(n, inv):
    return (n * inv) >> 64 if inv else n


def test_inverse_is_the_ceiling():
    for d in [2, 3, 5, 7, 64, 65, 1000, (1 << 16) + 1, (1 << 31) - 1, 1 << 31, (1 << 32) - 1]:
        assert udiv_inv(d) == -(-(1 << 64) // d)
        assert udiv_inv(d) < (1 << 64)  # fits the 64-bit word


def test_exhaustive_small():
    for d in range(1, 300):
        inv = udiv_inv(d)
        for n in range(0, 5000):
            assert udiv(n, inv) == n // d


def test_edges_and_random_32_bit():
    rng = np.random.default_rng(0)
    ds = [1, 2, 3, 6, 7, 8, 96, 97, 8192, 8193, 65535, 65536, 65537, 524287, 524288,
          (1 << 31) - 1, 1 << 31, (1 << 32) - 1]
    ds += [int(v) for v in rng.integers(1, 1 << 32, 200, dtype=np.uint64)]
    for d in ds:
        inv = udiv_inv(d)
        ns = [0, 1, d - 1, d, d + 1, 2 * d - 1, 2 * d, (1 << 31) - 1, (1 << 32) - 1]
        ns += [(k * d - 1) for k in (3, 1000, 65536) if k * d - 1 < (1 << 32)]
        ns += [int(v) for v in rng.integers(0, 1 << 32, 50, dtype=np.uint64)]
        for n in ns:
            if 0 <= n < (1 << 32):
                assert udiv(n, inv) == n // d, (n, d)


# ---- the inverse ZpR's segmented scan ---------------------------------------
# Each thread of the expansion kernel reduces its 16 symbols to (m, s): the
# number of end-of-block markers and the zigzag positions covered since its
# last marker (a literal covers 1, the run code eob - 17 + n covers n).  The
# pairs combine as (m1, s1) . (m2, s2) = (m1 + m2, s2 if m2 > 0 else s1 + s2);
# a parallel (Hillis-Steele) scan with this operator is only valid if it is
# associative.


def seg_cat(a, b):
    return (a[0] + b[0], b[1] if b[0] > 0 else a[1] + b[1])


def summarise(symbols, eob):
    m, s = 0, 0
    for x in symbols:
        if x == eob:
            m, s = m + 1, 0
        else:
            d = x - (eob - 16)
            s += d + 1 if 0 <= d < 16 else 1
    return m, s


def test_segment_combine_is_associative():
    dom = [(m, s) for m in range(3) for s in range(5)]
    for a in dom:
        for b in dom:
            for c in dom:
                assert seg_cat(seg_cat(a, b), c) == seg_cat(a, seg_cat(b, c))


def test_parallel_scan_equals_a_sequential_walk():
    eob = 272
    rng = np.random.default_rng(5)
    for trial in range(40):
        n_thr, per = 128, 16
        kinds = rng.random(n_thr * per)
        sym = np.where(kinds < 0.06, eob,
                       np.where(kinds < 0.25, rng.integers(eob - 16, eob, kinds.size),
                                rng.integers(-255, 256, kinds.size)))
        parts = [summarise(sym[t * per:(t + 1) * per], eob) for t in range(n_thr)]
        inc = list(parts)
        o = 1
        while o < n_thr:  # Hillis-Steele inclusive scan, as the warp shuffles do
            inc = [seg_cat(inc[t - o], inc[t]) if t >= o else inc[t] for t in range(n_thr)]
            o *= 2
        for t in range(n_thr):
            assert inc[t] == summarise(sym[:(t + 1) * per], eob)


# ---- the Huffman final decode's packed row descriptor -----------------------
# In the final decode each lane of a warp decodes one subsequence (consecutive
# subsequences on consecutive lanes) in rounds of up to 16 symbols; per round
# one shuffle carries ((o + done) - (o_0 + done_0)) << 5 | cap for the row a
# lane stores, o being the subsequence's output offset (an exclusive scan of
# the codeword counts, at most 256 per 256-bit subsequence) and done the
# symbols it has stored.  The offset must be non-negative and below 2^13
# (27 bits would still fit; 13 is the claim the kernel's comment makes).


def _rounds(counts, base=0):
    o = base + np.concatenate([[0], np.cumsum(counts)[:-1]])
    done = np.zeros_like(counts)
    worst, lo = 0, 0
    while np.any(done < counts):
        n = np.minimum(16, counts - done)
        rel = (o + done) - (o[0] + done[0])
        active = n > 0
        worst = max(worst, int(rel[active].max()))
        lo = min(lo, int(rel.min()))
        assert np.all(n <= 16) and np.all(n >= 0)
        done += n
    return worst, lo


def test_row_offsets_fit_the_packed_descriptor():
    rng = np.random.default_rng(9)
    cases = [np.full(32, 256), np.zeros(32, np.int64), np.r_[np.zeros(31, np.int64), 256],
             np.r_[1, np.full(31, 256)], np.r_[np.full(31, 256), 1]]
    cases += [rng.integers(0, 257, 32) for _ in range(2000)]
    cases += [np.where(rng.random(32) < 0.5, 0, rng.integers(200, 257, 32)) for _ in range(500)]
    worst = 0
    for c in cases:
        w, lo = _rounds(np.asarray(c, np.int64), base=int(rng.integers(0, 1 << 40)))
        assert lo >= 0
        worst = max(worst, w)
    assert worst <= 31 * 256 < 1 << 13


# ---- the inverse DCT's 8-point butterfly -------------------------------------
# The kernel's idct8 splits the orthonormal 8-point DCT-III into an even part
# E (frequencies 0, 2, 4, 6) and an odd part O (1, 3, 5, 7) with
# x[n] = E[n] + O[n] and x[7 - n] = E[n] - O[n], using the constants
# 0.5 cos(k pi / 16).  Restated here in fp64 and compared with scipy's
# orthonormal inverse DCT; the fp32 constants in the source are checked
# against the cosines.

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _idct8_butterfly(X, C):
    ee0, ee1 = C[4] * (X[0] + X[4]), C[4] * (X[0] - X[4])
    eo0, eo1 = C[2] * X[2] + C[6] * X[6], C[6] * X[2] - C[2] * X[6]
    e = [ee0 + eo0, ee1 + eo1, ee1 - eo1, ee0 - eo0]
    o = [C[1] * X[1] + C[3] * X[3] + C[5] * X[5] + C[7] * X[7],
         C[3] * X[1] - C[7] * X[3] - C[1] * X[5] - C[5] * X[7],
         C[5] * X[1] - C[1] * X[3] + C[7] * X[5] + C[3] * X[7],
         C[7] * X[1] - C[5] * X[3] + C[3] * X[5] - C[1] * X[7]]
    x = np.empty(8)
    for n in range(4):
        x[n], x[7 - n] = e[n] + o[n], e[n] - o[n]
    return x


def test_butterfly_is_the_orthonormal_inverse_dct():
    from scipy.fft import idct
    C = [0.5 * np.cos(k * np.pi / 16) for k in range(8)]
    rng = np.random.default_rng(3)
    for X in list(np.eye(8)) + [rng.standard_normal(8) for _ in range(200)]:
        assert np.allclose(_idct8_butterfly(X, C), idct(X, norm="ortho"), rtol=0, atol=1e-12)


def test_source_constants_are_the_cosines():
    src = open(os.path.join(ROOT, "paper_2609_09020_gb300", "csrc", "k_idct.cu")).read()
    got = dict((int(k), float(v)) for k, v in re.findall(r"kC(\d) = ([0-9.e+-]+)f", src))
    assert sorted(got) == list(range(1, 8))
    for k, v in got.items():
        assert np.float32(v) == np.float32(0.5 * np.cos(k * np.pi / 16)), k
    assert np.float32(got[4]) == np.float32(1 / np.sqrt(8))  # a(0), the DC scale
