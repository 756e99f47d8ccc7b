"""Integer index arithmetic of the inverse DCT kernel, restated and checked
on the CPU (no GPU).

Patch -> (image, plane row) uses division by invariant integers (Granlund &
Montgomery 1994): for 32-bit n and d, floor(n / d) = the high 64 bits of
n * inv with inv = ceil(2^64 / d), computed on the host as (2^64 - 1) // d + 1
(d == 1 stored as inv == 0, meaning n itself).  With inv d = 2^64 + e,
0 <= e < d, the product over 2^64 is n / d + n e / (d 2^64), and the error
term is below 2^-32 <= 1/d, so it never crosses the next integer.
"""
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
