"""The tensor-core kernel's cooperative upsampling, checked on the CPU for many
image widths (no GPU).

For each 128-pixel tile (origin x0) and level l >= 1, the kernel fills a
column buffer of NCOL(l) = 128/2^l + 4 entries with the level's columns
u_start + k, clamped into [0, W_l - 1], where u_start is the left tap of the
tile's first pixel; every pixel then interpolates horizontally between two
buffer entries.  Two index schemes pick those entries:

- generic: the pixel's own taps (computed in fp32 exactly as the kernel's
  bilinear_tap does) minus u_start, clamped into [0, NCOL - 1];
- fast (when W is a multiple of 2^(L-1)): tile-invariant relative taps
  floor((r + 1/2) / 2^l - 1/2) + 1 against u_start = x0/2^l - 1.

The clamp on buffer indices keeps every access in bounds whatever the
arithmetic does; these tests check that it never has to act, i.e. that the
buffer covers every tap, so that the horizontal pass equals the bilinear
definition (half-pixel centres, source coordinate clamped at 0, neighbour
clamped at W_l - 1) at every pixel of every tile.
"""
import numpy as np
import pytest

TILE = 128


def ncol(l):
    return (TILE >> l) + 4


def level_size(n, l):
    return -(-n // (1 << l))


def fma32(a, b, c):
    """fp32 fused multiply-add: the float64 a*b + c is exact for these
    operands (24-bit x 24-bit products, c = -1/2), then rounded once."""
    return (np.float64(a) * np.float64(b) + np.float64(c)).astype(np.float32)


def tap32(x, ratio32, n):
    """The kernel's bilinear_tap in fp32: (i0, i1, frac)."""
    s = np.maximum(fma32(np.asarray(x, np.float32) + np.float32(0.5), ratio32, -0.5), np.float32(0))
    i0 = s.astype(np.int64)  # truncation of a non-negative value
    return np.minimum(i0, n - 1), np.minimum(i0 + 1, n - 1), (s - i0.astype(np.float32))


def exact_taps(x, W, Wl):
    """The definition in exact rationals: s = max((x + 1/2) Wl / W - 1/2, 0)."""
    num = np.maximum((2 * np.asarray(x, np.int64) + 1) * Wl - W, 0)  # s = num / (2 W)
    i0 = num // (2 * W)
    return np.minimum(i0, Wl - 1), np.minimum(i0 + 1, Wl - 1), (num - i0 * 2 * W) / (2.0 * W)


def kernel_row(row, W, l, fast, ratio32):
    """The horizontal pass of every pixel of a W-wide image row at level l,
    tile by tile, as the kernel indexes its column buffer.  Returns the
    interpolated values and whether any buffer index had to be clamped."""
    Wl = row.size
    out = np.empty(W)
    clamped = False
    for x0 in range(0, W, TILE):
        r = np.arange(TILE)
        if fast:
            u_start = (x0 >> l) - 1
            sx = (r + 0.5) / (1 << l) - 0.5          # exact in fp32 (dyadic)
            fl = np.floor(sx)
            i0 = fl.astype(np.int64) + 1
            i1 = i0 + 1
            a = sx - fl
        else:
            u_start = int(tap32(x0, ratio32, Wl)[0])
            xc = np.minimum(x0 + r, W - 1)
            t0, t1, a = tap32(xc, ratio32, Wl)
            i0, i1 = t0 - u_start, t1 - u_start
        lim = ncol(l) - 1
        clamped |= bool(np.any((i0 < 0) | (i0 > lim) | (i1 < 0) | (i1 > lim)))
        i0, i1 = np.clip(i0, 0, lim), np.clip(i1, 0, lim)
        buf = row[np.clip(u_start + np.arange(ncol(l)), 0, Wl - 1)]
        v0, v1 = buf[i0], buf[i1]
        vals = v0 + a * (v1 - v0)
        n = min(TILE, W - x0)
        out[x0:x0 + n] = vals[:n]
    return out, clamped


WIDTHS = sorted(set(
    list(range(1, 300)) + [383, 511, 512, 513, 640, 767, 768, 769, 1000, 1023, 1024, 1025,
                           1919, 1920, 1921, 2047, 2048, 2049, 3839, 3840, 3841, 4095, 4097,
                           8191, 8193]))


@pytest.mark.parametrize("L", [2, 4, 7, 8, 12])
def test_buffer_covers_every_tap(L):
    rng = np.random.default_rng(L)
    for W in WIDTHS:
        fast = (L - 1 <= 7) and W % (1 << (L - 1)) == 0
        for l in range(1, L):
            Wl = level_size(W, l)
            ratio32 = np.float32(Wl / W)
            row = rng.standard_normal(Wl)
            got, clamped = kernel_row(row, W, l, fast, ratio32)
            assert not clamped, (W, L, l, fast)
            # the definition, exactly
            x = np.arange(W)
            e0, e1, ea = exact_taps(x, W, Wl)
            want = row[e0] + ea * (row[e1] - row[e0])
            # fp32 taps: ratio and coordinate each round once (<= 2^-24 of s + 1
            # each), so the value moves by at most 2^-23 (s + 1) times the
            # local slope; a wrong column would move it by O(1)
            slope = np.max(np.abs(np.diff(row))) if Wl > 1 else 0.0
            tol = 2.0 ** -22 * (Wl + 2) * slope + 1e-12
            assert np.max(np.abs(got - want)) <= tol, (W, L, l, fast)


def test_workload_widths_take_the_expected_scheme():
    # the decode workloads' widths are multiples of 2^(L-1) (256 = 2^8,
    # 768 = 3 x 2^8, 1920 = 15 x 2^7, 3840 = 30 x 2^7): the fast scheme; the
    # ragged test shapes take the generic one
    for W, L, fast in [(256, 4, True), (768, 7, True), (1920, 7, True), (3840, 8, True),
                       (131, 7, False), (383, 8, False), (200, 7, False), (1, 7, False)]:
        assert ((L - 1 <= 7) and W % (1 << (L - 1)) == 0) == fast
