"""Host-side checks of the C-ABI library: it builds for sm_103a, loads, and
exports every function include/pic_decode.h declares; size helpers and
argument checks answer without touching a GPU."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2609_09020_gb300 import build, pic
    build.build()
    return pic.load_library()


def declared_functions():
    names = []
    for fn in sorted(os.listdir(os.path.join(ROOT, "include"))):
        if fn.endswith(".h"):
            src = open(os.path.join(ROOT, "include", fn)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names += re.findall(r"\b(pic_\w+)\s*\(", src)
    return sorted(set(names))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("pic_decode_create", "pic_decode", "pic_decode_batch", "pic_decode_destroy",
                     "pic_status_string"):
        assert required in names


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name
        assert isinstance(getattr(lib, name), ctypes._CFuncPtr)


def test_size_helpers(lib):
    from paper_2609_09020_gb300 import pic, workloads as wk
    for wl in wk.WORKLOADS.values():
        assert pic.pic_latent_count(wl.H, wl.W, wl.L, wl.C) == wl.n_latents
        arch = pic.make_arch(wl.L, wl.C, wl.dims, wl.act)
        assert pic.pic_param_count(arch) == wl.n_params
    assert pic.pic_latent_count(0, 5, 1, 1) == -1


def test_status_strings(lib):
    from paper_2609_09020_gb300 import pic
    for s in (0, -1, -2, -3, -4, -5):
        assert pic.pic_status_string(s) not in ("", "unknown status")
    assert pic.pic_status_string(7) == "unknown status"


def test_null_and_bad_arguments_are_rejected_without_a_gpu(lib):
    from paper_2609_09020_gb300 import pic
    assert lib.pic_decode(None, None, None, None, 4, 4, None, None) == pic.PIC_ERR_INVALID_ARG
    assert lib.pic_decode_batch(None, 1, None, None, None, 4, 4, None, None) == pic.PIC_ERR_INVALID_ARG
    assert lib.pic_decode_batch_host(None, 1, None, None, None, 4, 4, None, None) == pic.PIC_ERR_INVALID_ARG
    assert lib.pic_decode_check(None, None) == pic.PIC_ERR_INVALID_ARG
    lib.pic_decode_destroy(None)
    assert pic.pic_decode_kernel_name(None) == ""
    h = ctypes.c_void_p(123)
    assert lib.pic_decode_create(None, ctypes.byref(h)) == pic.PIC_ERR_INVALID_ARG
    assert h.value is None
    bad = pic.make_arch(2, 1, (3, 8, 3))          # dims[0] != L*C
    assert lib.pic_decode_create(ctypes.byref(bad), ctypes.byref(h)) == pic.PIC_ERR_INVALID_ARG
    wide = pic.make_arch(2, 1, (2, 256, 3), max_H=4, max_W=4)   # width above the envelope
    assert lib.pic_decode_create(ctypes.byref(wide), ctypes.byref(h)) == pic.PIC_ERR_UNSUPPORTED


def test_create_without_gpu_fails_cleanly(lib):
    torch = pytest.importorskip("torch")
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    from paper_2609_09020_gb300 import pic
    arch = pic.make_arch(4, 1, (4, 16, 16, 3), max_H=8, max_W=8)
    h = ctypes.c_void_p()
    rc = lib.pic_decode_create(ctypes.byref(arch), ctypes.byref(h))
    assert rc in (pic.PIC_ERR_UNSUPPORTED, pic.PIC_ERR_CUDA) and h.value is None


def test_izpr_workspace_and_argument_checks(lib):
    from paper_2609_09020_gb300 import pic
    assert pic.pic_izpr_workspace_bytes(-1) == -1
    assert pic.pic_izpr_workspace_bytes(0) == 32
    assert pic.pic_izpr_workspace_bytes(1) >= 32 + 4 + 8
    # a status word and total, then per 2048-symbol chunk its offset in its
    # group (int32), per group of 8 chunks its count (int32) and base (int64)
    n = 10 ** 8
    chunks = -(-n // 2048)
    groups = -(-chunks // 8)
    assert pic.pic_izpr_workspace_bytes(n) >= 32 + 4 * chunks + 12 * groups
    # rejected before any CUDA call
    assert pic.pic_izpr_decode(None, 10, 30, 1, None, None, None, 0, None) == pic.PIC_ERR_INVALID_ARG
    assert pic.pic_izpr_decode(None, -1, 30, 1, None, None, None, 0, None) == pic.PIC_ERR_INVALID_ARG
    assert pic.pic_izpr_status(None, None) == pic.PIC_ERR_INVALID_ARG


def test_idct_block_count_and_argument_checks(lib, orc):
    from paper_2609_09020_gb300 import pic
    from paper_2609_09020_gb300 import workloads as wk
    for H, W, L, C in [(512, 768, 7, 1), (1080, 1920, 7, 2), (5, 3, 4, 4), (1, 1, 1, 1),
                       (2160, 3840, 8, 2)]:
        n = pic.pic_idct_block_count(H, W, L, C)
        assert n == orc.block_count(H, W, L, C) == wk.block_count(H, W, L, C)
    assert pic.pic_idct_block_count(0, 5, 1, 1) == -1
    assert pic.pic_idct_block_count(5, 5, 13, 1) == -1
    assert pic.pic_idct_block_count(5, 5, 1, 5) == -1
    # rejected before any CUDA call
    assert pic.pic_idct_unpatchify(None, None, 1, 8, 8, 1, 1, None, None) == pic.PIC_ERR_INVALID_ARG
    assert pic.pic_idct_unpatchify(16, 16, 0, 8, 8, 1, 1, 16, None) == pic.PIC_ERR_INVALID_ARG
    assert pic.pic_idct_unpatchify(8, 16, 1, 8, 8, 1, 1, 16, None) == pic.PIC_ERR_INVALID_ARG


def test_fp32_latent_arch_is_validated(lib):
    """latent_format outside the enum is refused at create (no device needed
    to reach that check)."""
    from paper_2609_09020_gb300 import pic
    a = pic.make_arch(2, 1, [2, 8, 3], max_H=8, max_W=8, latent=2)
    h = pic._P()
    assert lib.pic_decode_create(pic.ctypes.byref(a), pic.ctypes.byref(h)) == pic.PIC_ERR_UNSUPPORTED


def test_fuse_modulation_argument_checks(lib):
    from paper_2609_09020_gb300 import pic
    a = pic.make_arch(7, 1, [7, 64, 64, 3], max_H=8, max_W=8)
    assert pic.pic_fuse_modulation(a, 1, None, None, None) == pic.PIC_ERR_INVALID_ARG
    assert pic.pic_fuse_modulation(a, 0, 16, 16, 16) == pic.PIC_ERR_INVALID_ARG
    assert pic.pic_fuse_modulation(a, 1, 16, 16, 8) == pic.PIC_ERR_INVALID_ARG  # misaligned out
    one = pic.make_arch(7, 1, [7, 3], max_H=8, max_W=8)  # no MLP^s to fuse after
    assert pic.pic_fuse_modulation(one, 1, 16, 16, 16) == pic.PIC_ERR_INVALID_ARG


def test_output_format_is_validated(lib):
    from paper_2609_09020_gb300 import pic
    a = pic.make_arch(2, 1, [2, 8, 3], max_H=8, max_W=8, output=3)
    h = pic._P()
    assert lib.pic_decode_create(pic.ctypes.byref(a), pic.ctypes.byref(h)) == pic.PIC_ERR_UNSUPPORTED


def test_huffman_workspace_and_argument_checks(lib):
    from paper_2609_09020_gb300 import pic
    assert pic.pic_huffman_workspace_bytes(8, 1, 12) > 0
    assert pic.pic_huffman_workspace_bytes(7, 1, 12) == -1   # not whole subsequences
    assert pic.pic_huffman_workspace_bytes(8, 1, 13) == -1   # precision above 12
    assert pic.pic_huffman_decode(None, 8, None, None, 1, None, None, 4, 12, None, None, None, 0,
                                  None) == pic.PIC_ERR_INVALID_ARG
    assert pic.pic_huffman_status(None, None) == pic.PIC_ERR_INVALID_ARG


def test_fma_peak_helper_without_gpu(lib):
    """The FMA microbenchmark's flop count and argument checks (include/pic_measure.h)."""
    from paper_2609_09020_gb300 import pic
    assert pic.load_library().pic_fma_peak_flops(0, 1) == -1
    assert pic.load_library().pic_fma_peak_flops(1, 0) == -1
    assert pic.load_library().pic_fma_peak_flops(2, 3) == 2 * 256 * 3 * 16 * 8 * 2
    assert pic.load_library().pic_fma_peak_launch(None, 1, 1, None) == pic.PIC_ERR_INVALID_ARG


def test_noalloc_entry_and_size_helpers_reject_bad_arguments(lib):
    """pic_decode_batch_noalloc validates the arch before touching a device;
    the size helpers answer -1 outside their domain."""
    from paper_2609_09020_gb300 import pic
    p = ctypes.c_void_p(256)
    assert lib.pic_decode_batch_noalloc(None, 1, p, p, p, 8, 8, p, None) == pic.PIC_ERR_INVALID_ARG
    bad = pic.make_arch(2, 1, (3, 8, 3), max_H=8, max_W=8)           # dims[0] != L*C
    assert lib.pic_decode_batch_noalloc(ctypes.byref(bad), 1, p, p, p, 8, 8, p,
                                        None) == pic.PIC_ERR_INVALID_ARG
    wide = pic.make_arch(2, 1, (2, 256, 3), max_H=8, max_W=8)        # width above the envelope
    assert lib.pic_decode_batch_noalloc(ctypes.byref(wide), 1, p, p, p, 8, 8, p,
                                        None) == pic.PIC_ERR_UNSUPPORTED
    staged = pic.make_arch(2, 1, (2, 16, 3), max_H=8, max_W=8, staging=3)  # no such staging
    assert lib.pic_decode_batch_noalloc(ctypes.byref(staged), 1, p, p, p, 8, 8, p,
                                        None) == pic.PIC_ERR_UNSUPPORTED
    assert lib.pic_param_count(None) == -1
    assert pic.pic_latent_count(8, 8, 31, 1) == -1 and pic.pic_latent_count(8, 8, 1, 0) == -1
    assert pic.pic_latent_count(1, 1, 30, 4) == 30 * 4   # every level of a 1x1 image is 1x1
