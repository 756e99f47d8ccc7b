"""GPU Huffman decoding (Sec. 3.3; self-synchronising parallel decoding as
in GPUHD) against the oracle's bit-by-bit canonical decoder, bit-exact,
through the C ABI."""
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


def _pack_batch(streams, p):
    """Per-stream (tab_value, tab_len, words, n_bits) -> batch arrays."""
    B = len(streams)
    mt = max(1, max(len(s[0]) for s in streams))
    tv = np.zeros((B, mt), np.int32)
    tl = np.zeros((B, mt), np.int32)
    for b, (v, ln, _, _) in enumerate(streams):
        tv[b, :len(v)] = v
        tl[b, :len(ln)] = ln
    word_off = np.r_[0, np.cumsum([len(s[2]) for s in streams])].astype(np.int64)
    return dict(words=np.concatenate([s[2] for s in streams]).astype(np.uint32), word_off=word_off,
                n_bits=np.array([s[3] for s in streams], np.int64), tab_value=tv, tab_len=tl, p=p)


def _gpu(d, sym_off, check=True):
    import torch
    from paper_2609_09020_gb300 import pic
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    out = pic.huffman_decode(t(d["words"].view(np.int32)), t(d["word_off"]), t(d["n_bits"]),
                             t(d["tab_value"]), t(d["tab_len"]), d["p"], t(sym_off), check=check)
    return out.cpu().numpy()


def test_full_batch_against_oracle(orc):
    """The 64-image batch's ZpR streams (26 M symbols, 64 tables) in one
    call; images 0, 17 and 63 also through the oracle's decoder."""
    h = wk.huffman_streams("c5")
    got = _gpu(h, h["sym_off"])
    assert np.array_equal(got, h["symbols"])
    for b in (0, 17, 63):
        w = h["words"][h["word_off"][b]:h["word_off"][b + 1]]
        n = h["tab_len"][b].astype(bool).sum()
        ref = orc.huffman_decode(w, h["n_bits"][b], h["tab_value"][b, :n], h["tab_len"][b, :n],
                                 int(h["sym_off"][b + 1] - h["sym_off"][b]))
        assert np.array_equal(got[h["sym_off"][b]:h["sym_off"][b + 1]], ref), b


@pytest.mark.parametrize("p", [4, 7, 12])
def test_edge_streams(orc, p):
    """Single-symbol codes (one 1-bit codeword), an empty stream, streams of
    1, 2 and 300 symbols, codes near the precision, long streams."""
    rng = np.random.Generator(np.random.PCG64(p))
    cases = [np.full(1, 5, np.int32), np.zeros(0, np.int32), np.array([3, -3], np.int32),
             np.full(1000, -7, np.int32),
             rng.integers(-(2 ** (p - 1)), 2 ** (p - 1), 300).astype(np.int32),
             np.clip(np.rint(rng.laplace(0, 2.0 ** (p - 3), 20000)), 1 - 2 ** (p - 1),
                     2 ** (p - 1) - 1).astype(np.int32)]
    streams, syms = [], []
    for s in cases:
        if s.size == 0:
            streams.append((np.array([1], np.int32), np.array([1], np.int32),
                            np.zeros(wk.HUFF_WORDS_PER_SUBSEQ, np.uint32), 0))
        else:
            streams.append(wk.huffman_pack(s, p))
        syms.append(s)
    d = _pack_batch(streams, p)
    sym_off = np.r_[0, np.cumsum([s.size for s in syms])].astype(np.int64)
    got = _gpu(d, sym_off)
    assert np.array_equal(got, np.concatenate(syms))


def test_full_range_values():
    """Symbol values anywhere in int32 (the lookup tables hold a symbol's
    row in the stored table, not its value)."""
    rng = np.random.Generator(np.random.PCG64(31))
    alphabet = np.array([-2 ** 31, 2 ** 31 - 1, 2 ** 30, -2 ** 29 + 7, 0, 5, -(2 ** 23), 2 ** 23],
                        np.int64).astype(np.int32)
    s = alphabet[rng.integers(0, alphabet.size, 5000)]
    d = _pack_batch([wk.huffman_pack(s, 12)], 12)
    got = _gpu(d, np.array([0, s.size], np.int64))
    assert np.array_equal(got, s)


def test_malformed_streams_are_flagged():
    from paper_2609_09020_gb300 import pic
    rng = np.random.Generator(np.random.PCG64(97))
    s = np.rint(rng.laplace(0, 3, 2000)).astype(np.int32)
    v, ln, w, nb = wk.huffman_pack(s, 12)
    sym_off = np.array([0, s.size], np.int64)
    good = _pack_batch([(v, ln, w, nb)], 12)
    assert np.array_equal(_gpu(good, sym_off), s)
    bad_count = np.array([0, s.size + 1], np.int64)
    truncated = _pack_batch([(v, ln, w, nb - 1)], 12)           # last codeword cut short
    kraft = _pack_batch([(v, np.maximum(ln - 1, 1), w, nb)], 12)  # lengths too short for a code
    for d, so in ((good, bad_count), (truncated, sym_off), (kraft, sym_off)):
        with pytest.raises(pic.PicError):
            _gpu(d, so)
    # an incomplete code (one symbol: codeword "0") meets a "1" bit
    one = _pack_batch([(np.array([4], np.int32), np.array([1], np.int32),
                        np.r_[np.uint32(0x40000000), np.zeros(7, np.uint32)], 3)], 5)
    with pytest.raises(pic.PicError):
        _gpu(one, np.array([0, 3], np.int64))
