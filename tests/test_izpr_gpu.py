"""GPU inverse ZpR (Algorithm 1 + marker compaction) against the fp64-free
integer oracle: bit-exact coefficients and offsets, through the C ABI."""
import numpy as np
import pytest

from paper_2609_09020_gb300 import workloads as wk

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_09020_gb300 import build
    build.build()


def _gpu(stream_np, eob, n_blocks):
    import torch
    from paper_2609_09020_gb300 import pic
    sym = torch.from_numpy(np.ascontiguousarray(stream_np, dtype=np.int32)).to("cuda:0")
    c, o = pic.izpr_decode(sym, eob, n_blocks)
    return c.cpu().numpy(), o.cpu().numpy()


def _roundtrip(orc, blocks, eob=None):
    eob = int(np.abs(blocks).max()) + 17 if eob is None else eob
    s = orc.zpr_encode(blocks, eob)
    c, o = _gpu(s, eob, blocks.shape[0])
    assert np.array_equal(c, blocks)
    assert np.array_equal(c, orc.izpr(s, eob, blocks.shape[0]))
    assert np.array_equal(o, np.nonzero(s == eob)[0])
    return s


def test_hand_stream(orc):
    import oracle_pins
    g = oracle_pins.load_golden("zpr_blocks.txt")
    blocks = oracle_pins._golden_blocks(g)
    stream = np.array([int(v) for v in g["stream"]], dtype=np.int32)
    c, o = _gpu(stream, int(g["eob"][0]), blocks.shape[0])
    assert np.array_equal(c, blocks)
    assert o.tolist() == [11, 12, 14]


@pytest.mark.parametrize("n,seed", [(1, 0), (7, 1), (4000, 2), (33333, 3)])
def test_random_blocks(orc, n, seed):
    _roundtrip(orc, wk.dct_blocks(n, seed))


def test_edge_blocks(orc):
    rng = np.random.Generator(np.random.PCG64(5))
    b = np.zeros((9, 64), np.int32)
    b[1] = rng.integers(1, 100, 64)          # 64 literals, no zeros
    b[2, 63] = -7                            # 63-zero prefix: 16+16+16+15
    b[3, 0] = 1
    b[4, ::2] = 3                            # alternating single zeros
    b[5, 1:] = -1                            # leading zero then 63 literals
    b[7] = rng.integers(-2, 3, 64)
    _roundtrip(orc, b)
    _roundtrip(orc, b, eob=1000)             # any eob above the literals + 16


def test_unaligned_stream(orc):
    """Symbols starting 4 bytes past a 16-byte boundary (the scalar load path)."""
    import torch
    from paper_2609_09020_gb300 import pic
    blocks = wk.dct_blocks(3000, 21)
    eob = int(np.abs(blocks).max()) + 17
    s = orc.zpr_encode(blocks, eob)
    padded = torch.from_numpy(np.r_[np.int32(0), s].astype(np.int32)).to("cuda:0")
    c, o = pic.izpr_decode(padded[1:], eob, blocks.shape[0])
    assert padded[1:].data_ptr() % 16 != 0
    assert np.array_equal(c.cpu().numpy(), blocks)
    assert np.array_equal(o.cpu().numpy(), np.nonzero(s == eob)[0])


def test_all_zero_blocks(orc):
    """Every block empty: one marker per symbol, so every chunk holds as many
    blocks as symbols (many expansion passes per chunk)."""
    _roundtrip(orc, np.zeros((10000, 64), np.int32))


def test_eob_zero(orc):
    """eob = 0: the zeros past the end of the stream must not count as markers."""
    rng = np.random.Generator(np.random.PCG64(9))
    b = np.where(rng.random((777, 64)) < 0.3, rng.integers(-300, -17, (777, 64)), 0).astype(np.int32)
    _roundtrip(orc, b, eob=0)


def test_empty_stream():
    c, o = _gpu(np.zeros(0, np.int32), 40, 0)
    assert c.shape == (0, 64) and o.shape == (0,)


def test_full_size_batch(orc):
    """A batch's worth of blocks: the 64 Kodak-sized latent pyramids of the
    throughput workload hold ~8,200 blocks each."""
    _roundtrip(orc, wk.dct_blocks(64 * 8192, 11))


def test_malformed_streams_are_flagged():
    import torch
    from paper_2609_09020_gb300 import pic
    eob = 30
    cases = [
        (np.array([29, 29, 29, 29, 29, 30], np.int32), 1),   # 80 positions in one block
        (np.array([1, 30, 2, 30], np.int32), 3),             # fewer markers than blocks
        (np.array([1, 30, 2, 30, 30], np.int32), 2),         # more markers than blocks
        (np.array([31, 30], np.int32), 1),                   # value above eob
        (np.array([1, 30, 5], np.int32), 1),                 # symbols after the last marker
        (np.zeros(0, np.int32), 2),                          # no symbols, two blocks expected
        (np.r_[np.full(70, 3), 30].astype(np.int32), 1),     # 70 literals in one block
        (np.r_[np.full(5000, 3), 30].astype(np.int32), 1),   # a block across a whole chunk
    ]
    for s, n in cases:
        with pytest.raises(pic.PicError):
            _gpu(s, eob, n)
