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


# ---- TMA staging (the TMA-staged kernels).  Per tile, the group's issuing
# warp loads every (level, channel, row) segment as one box of a 1-D tensor
# map over the call's latent words: level 0 the tile's 128 words of row y,
# level l >= 1 the words u_start .. u_start + NCOL(l) - 1 of rows i0 and i1 of
# the tile row's vertical tap.  A box starts at the segment's first word s
# rounded down to a multiple of 4 (TMA's 16-byte rule), so column k of the
# segment is box word (s & 3) + k.

def box_w(l):
    """tma_box_w of the kernels: level 0 128 + 4 words; level l >= 1 NCOL(l)
    + 3 rounded up to a multiple of 4."""
    return TILE + 4 if l == 0 else -(-(ncol(l) + 3) // 4) * 4


def test_box_widths():
    assert [box_w(l) for l in range(10)] == [132, 72, 40, 24, 16, 12, 12, 8, 8, 8]
    assert all(box_w(l) % 4 == 0 and box_w(l) <= 256 for l in range(13))
    # the largest in-box index a read can take: 3 + (segment length - 1)
    assert 3 + TILE - 1 < box_w(0)
    assert all(3 + ncol(l) - 1 < box_w(l) for l in range(1, 13))


@pytest.mark.parametrize("L", [2, 4, 7, 8, 12])
def test_tma_segment_columns_stay_inside_the_box(L):
    """The column the vertical pass reads, clamp(u_start + i, 0, W_l - 1) -
    u_start, lies in [0, NCOL(l)) for every item i of every tile, both tap
    schemes, so (s & 3) + column stays inside the box."""
    for W in WIDTHS:
        fast = (L - 1 <= 7) and W % (1 << (L - 1)) == 0
        for l in range(1, L):
            Wl = level_size(W, l)
            ratio32 = np.float32(Wl / W)
            for x0 in range(0, W, TILE):
                u_start = (x0 >> l) - 1 if fast else int(tap32(x0, ratio32, Wl)[0])
                assert u_start >= -1
                col = np.clip(u_start + np.arange(ncol(l)), 0, Wl - 1) - u_start
                assert col.min() >= 0 and col.max() < ncol(l), (W, L, l, x0)
                for s in range(4):  # any alignment of the segment start
                    assert (s & 3) + col.max() < box_w(l)


def test_tma_box_reads_the_defined_words():
    """Words s & ~3 .. of a buffer, read at (s & 3) + k, are words s + k: a
    tile's segments come back whatever the alignment of their start,
    including segments that begin one word before a row (u_start = -1,
    never read: the clamp takes column 0) and segments at the buffer's end
    (zero fill past it, never read either)."""
    rng = np.random.default_rng(3)
    buf = rng.integers(-63, 64, 1000)
    for s in list(range(0, 40)) + [995, 996, 999]:
        for bw in (8, 12, 72, 132):
            x = s & ~3
            box = np.array([buf[x + k] if x + k < buf.size else 0 for k in range(bw)])
            n = min(bw - 3, buf.size - s)
            assert np.array_equal(box[(s & 3) + np.arange(n)], buf[s:s + n])


@pytest.mark.parametrize("L,C", [(4, 1), (7, 1), (8, 2), (12, 4)])
def test_tma_boxes_and_slots(L, C):
    """The issuing warp's lane q -> (level, channel, row) map hits every
    segment of a tile exactly once, and the segments' slots in a buffer are
    disjoint, start on 128 bytes (a tiled TMA copy's shared-memory
    destination), hold their box and fill the buffer (TmaSlots)."""
    rows = lambda l: 1 if l == 0 else 2
    slot = lambda l: -(-box_w(l) * 4 // 128) * 128
    def off(l, c, r):
        o = sum(C * rows(k) * slot(k) for k in range(l))
        return o + (c * rows(l) + r) * slot(l)
    n = C * (2 * L - 1)
    seen = []
    for q in range(n):
        if q < C:
            l, c, r = 0, q, 0
        else:
            q2 = q - C
            l, c, r = 1 + q2 // (2 * C), (q2 >> 1) % C, q2 & 1
        assert 0 <= l < L and 0 <= c < C and r < rows(l)
        seen.append((l, c, r))
    assert len(set(seen)) == n == sum(C * rows(l) for l in range(L))
    spans = sorted((off(l, c, r), off(l, c, r) + slot(l), box_w(l) * 4) for l, c, r in seen)
    assert all(a % 128 == 0 and box <= e - a for a, e, box in spans)
    assert all(spans[k][1] == spans[k + 1][0] for k in range(n - 1))
    assert spans[0][0] == 0 and spans[-1][1] == off(L, 0, 0)


# ---- Per-warp column buffers.  Each warp of a group (its 32 consecutive
# pixels, offset xo = 32 w within the 128-pixel tile) fills its own column
# buffer of NCOLW(l) = 32/2^l + 4 entries from its own left tap, so no
# barrier across the group's warps is needed: the fast scheme's relative taps
# use the pixel's offset within a 2^l-aligned span, (xo mod 2^l) + lane,
# which is tile-invariant because the tile origin is a multiple of 128.
SEG = 32


def ncolw(l):
    return (SEG >> l) + 4


def warp_row(row, W, l, fast, ratio32):
    """The horizontal pass of every pixel of a W-wide row at level l, warp by
    warp, as the kernel indexes each warp's column buffer; returns the values
    and whether any buffer index had to be clamped."""
    Wl = row.size
    out = np.empty(W)
    clamped = False
    for x0 in range(0, W, TILE):
        for xo in range(0, TILE, SEG):
            X = x0 + xo
            lane = np.arange(SEG)
            if fast:
                u_start = (X >> l) - 1
                sx = (((xo % (1 << l)) + lane) + 0.5) / (1 << l) - 0.5  # exact (dyadic)
                fl = np.floor(sx)
                i0 = fl.astype(np.int64) + 1
                i1 = i0 + 1
                a = sx - fl
            else:
                u_start = int(tap32(X, ratio32, Wl)[0])
                xc = np.minimum(X + lane, W - 1)
                t0, t1, a = tap32(xc, ratio32, Wl)
                i0, i1 = t0 - u_start, t1 - u_start
            lim = ncolw(l) - 1
            valid = X + lane < W  # pixels past the row's end are never stored
            bad = (i0 < 0) | (i0 > lim) | (i1 < 0) | (i1 > lim)
            clamped |= bool(np.any(bad & valid))
            i0, i1 = np.clip(i0, 0, lim), np.clip(i1, 0, lim)
            buf = row[np.clip(u_start + np.arange(ncolw(l)), 0, Wl - 1)]
            vals = buf[i0] + a * (buf[i1] - buf[i0])
            n = max(0, min(SEG, W - X))
            out[X:X + n] = vals[:n]
    return out, clamped


@pytest.mark.parametrize("L", [2, 4, 7, 8, 12])
def test_warp_buffers_cover_every_tap(L):
    rng = np.random.default_rng(100 + L)
    for W in WIDTHS:
        fast = (L - 1 <= 7) and W % (1 << (L - 1)) == 0
        for l in range(1, L):
            Wl = level_size(W, l)
            ratio32 = np.float32(Wl / W)
            row = rng.standard_normal(Wl)
            got, clamped = warp_row(row, W, l, fast, ratio32)
            assert not clamped, (W, L, l, fast)
            x = np.arange(W)
            e0, e1, ea = exact_taps(x, W, Wl)
            want = row[e0] + ea * (row[e1] - row[e0])
            slope = np.max(np.abs(np.diff(row))) if Wl > 1 else 0.0
            tol = 2.0 ** -22 * (Wl + 2) * slope + 1e-12
            assert np.max(np.abs(got - want)) <= tol, (W, L, l, fast)
