"""ctypes binding of the C ABI in include/pic_decode.h (libpic_gb300.so).

Argument marshalling only: every step of the decode runs in the library's CUDA
kernels.  The functions keep the C names; ``Decoder`` wraps a handle and
accepts torch CUDA tensors (PyTorch supplies device memory and streams) or,
for ``decode_batch_host``, host numpy arrays, and checks each buffer's size,
contiguity and device before the call (the C ABI sees bare pointers).

Loading fails loudly (ImportError/OSError) when the library has not been
built; there is no CPU fallback.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from . import build as _build

PIC_OK = 0
PIC_ERR_INVALID_ARG = -1
PIC_ERR_UNSUPPORTED = -2
PIC_ERR_CUDA = -3
PIC_ERR_ALLOC = -4
PIC_ERR_TIMEOUT = -5

PIC_ACT_RELU = 0
PIC_ACT_GELU = 1
PIC_PREC_FP32 = 0
PIC_PREC_FP16_TC = 1
PIC_PREC_FP16_TC_LO8 = 2
PIC_LATENT_INT32 = 0
PIC_LATENT_FP32 = 1

ACTS = {"relu": PIC_ACT_RELU, "gelu": PIC_ACT_GELU}
PRECS = {"fp32": PIC_PREC_FP32, "fp16_tc": PIC_PREC_FP16_TC, "fp16_tc_lo8": PIC_PREC_FP16_TC_LO8}
LATENTS = {"int32": PIC_LATENT_INT32, "fp32": PIC_LATENT_FP32}
PIC_OUT_F32_CHW = 0
PIC_OUT_F32_HWC = 1
PIC_OUT_U8_HWC = 2
OUTPUTS = {"f32_chw": PIC_OUT_F32_CHW, "f32_hwc": PIC_OUT_F32_HWC, "u8_hwc": PIC_OUT_U8_HWC}
PIC_STAGING_AUTO, PIC_STAGING_COPIES, PIC_STAGING_TMA = 0, 1, 2
STAGINGS = {"auto": PIC_STAGING_AUTO, "copies": PIC_STAGING_COPIES, "tma": PIC_STAGING_TMA}


class pic_arch(ctypes.Structure):
    _fields_ = [
        ("num_levels", ctypes.c_int),
        ("channels_per_level", ctypes.c_int),
        ("num_layers", ctypes.c_int),
        ("dims", ctypes.c_int * 7),
        ("hidden_act", ctypes.c_int),
        ("precision", ctypes.c_int),
        ("clamp_output", ctypes.c_int),
        ("max_H", ctypes.c_int),
        ("max_W", ctypes.c_int),
        ("max_batch", ctypes.c_int),
        ("latent_format", ctypes.c_int),
        ("output_format", ctypes.c_int),
        ("staging", ctypes.c_int),
    ]


_P = ctypes.c_void_p
_lib = None


def library_path() -> str:
    return _build.LIB


def load_library():
    """Loads libpic_gb300.so (built by ``build.build()``); raises if missing."""
    global _lib
    if _lib is not None:
        return _lib
    path = library_path()
    if not os.path.exists(path):
        raise ImportError(f"{path} is missing: run paper_2609_09020_gb300.build.build() first "
                          "(there is no CPU fallback)")
    lib = ctypes.CDLL(path)
    i, i64 = ctypes.c_int, ctypes.c_int64
    lib.pic_decode_create.argtypes = [ctypes.POINTER(pic_arch), ctypes.POINTER(_P)]
    lib.pic_decode_create.restype = i
    lib.pic_decode.argtypes = [_P, _P, _P, _P, i, i, _P, _P]
    lib.pic_decode.restype = i
    lib.pic_decode_batch.argtypes = [_P, i, _P, _P, _P, i, i, _P, _P]
    lib.pic_decode_batch.restype = i
    lib.pic_decode_batch_host.argtypes = [_P, i, _P, _P, _P, i, i, _P, _P]
    lib.pic_decode_batch_host.restype = i
    lib.pic_decode_batch_noalloc.argtypes = [ctypes.POINTER(pic_arch), i, _P, _P, _P, i, i, _P, _P]
    lib.pic_decode_batch_noalloc.restype = i
    lib.pic_decode_noalloc_check.argtypes = [_P]
    lib.pic_decode_noalloc_check.restype = i
    lib.pic_decode_test_wait_fault.argtypes = [i, ctypes.c_uint]
    lib.pic_decode_test_wait_fault.restype = i
    lib.pic_decode_check.argtypes = [_P, _P]
    lib.pic_decode_check.restype = i
    lib.pic_decode_destroy.argtypes = [_P]
    lib.pic_decode_destroy.restype = None
    lib.pic_decode_kernel_name.argtypes = [_P]
    lib.pic_decode_kernel_name.restype = ctypes.c_char_p
    lib.pic_latent_count.argtypes = [i, i, i, i]
    lib.pic_latent_count.restype = i64
    lib.pic_param_count.argtypes = [ctypes.POINTER(pic_arch)]
    lib.pic_param_count.restype = i64
    lib.pic_izpr_workspace_bytes.argtypes = [i64]
    lib.pic_izpr_workspace_bytes.restype = i64
    lib.pic_izpr_decode.argtypes = [_P, i64, ctypes.c_int32, i64, _P, _P, _P, ctypes.c_size_t, _P]
    lib.pic_izpr_decode.restype = i
    lib.pic_izpr_status.argtypes = [_P, _P]
    lib.pic_izpr_status.restype = i
    lib.pic_idct_block_count.argtypes = [i, i, i, i]
    lib.pic_idct_block_count.restype = i64
    lib.pic_idct_unpatchify.argtypes = [_P, _P, i, i, i, i, i, _P, _P]
    lib.pic_idct_unpatchify.restype = i
    lib.pic_fuse_modulation.argtypes = [ctypes.POINTER(pic_arch), i, _P, _P, _P, _P]
    lib.pic_fuse_modulation.restype = i
    lib.pic_huffman_workspace_bytes.argtypes = [i64, i, i]
    lib.pic_huffman_workspace_bytes.restype = i64
    lib.pic_huffman_decode.argtypes = [_P, i64, _P, _P, i, _P, _P, i, i, _P, _P, _P,
                                       ctypes.c_size_t, _P]
    lib.pic_huffman_decode.restype = i
    lib.pic_huffman_status.argtypes = [_P, _P]
    lib.pic_huffman_status.restype = i
    lib.pic_fma_peak_flops.argtypes = [i, i]
    lib.pic_fma_peak_flops.restype = i64
    lib.pic_fma_peak_launch.argtypes = [_P, i, i, _P]
    lib.pic_fma_peak_launch.restype = i
    lib.pic_status_string.argtypes = [i]
    lib.pic_status_string.restype = ctypes.c_char_p
    _lib = lib
    return lib


class PicError(RuntimeError):
    def __init__(self, status: int, where: str):
        lib = load_library()
        super().__init__(f"{where}: {lib.pic_status_string(status).decode()} ({status})")
        self.status = status


def make_arch(L, C, dims, act="relu", precision="fp32", clamp=True, max_H=1, max_W=1,
              max_batch=1, latent="int32", output="f32_chw", staging="auto") -> pic_arch:
    a = pic_arch()
    a.num_levels, a.channels_per_level, a.num_layers = L, C, len(dims) - 1
    for k, d in enumerate(dims):
        a.dims[k] = int(d)
    a.hidden_act = ACTS[act] if isinstance(act, str) else int(act)
    a.precision = PRECS[precision] if isinstance(precision, str) else int(precision)
    a.clamp_output = int(bool(clamp))
    a.max_H, a.max_W, a.max_batch = max_H, max_W, max_batch
    a.latent_format = LATENTS[latent] if isinstance(latent, str) else int(latent)
    a.output_format = OUTPUTS[output] if isinstance(output, str) else int(output)
    a.staging = STAGINGS[staging] if isinstance(staging, str) else int(staging)
    return a


# ---- the C functions, same names -------------------------------------------
def pic_decode_create(arch: pic_arch) -> int:
    h = _P()
    rc = load_library().pic_decode_create(ctypes.byref(arch), ctypes.byref(h))
    if rc != PIC_OK:
        raise PicError(rc, "pic_decode_create")
    return h.value


def pic_decode(h, latents, steps, weights, H, W, out_rgb, stream=None) -> int:
    return load_library().pic_decode(h, latents, steps, weights, H, W, out_rgb, stream)


def pic_decode_batch(h, B, latents, steps, weights, H, W, out_rgb, stream=None) -> int:
    return load_library().pic_decode_batch(h, B, latents, steps, weights, H, W, out_rgb, stream)


def pic_decode_batch_host(h, B, latents, steps, weights, H, W, out_rgb, stream=None) -> int:
    return load_library().pic_decode_batch_host(h, B, latents, steps, weights, H, W, out_rgb,
                                                stream)


def pic_decode_batch_noalloc(arch: pic_arch, B, latents, steps, weights, H, W, out_rgb,
                             stream=None) -> int:
    return load_library().pic_decode_batch_noalloc(ctypes.byref(arch), B, latents, steps, weights,
                                                   H, W, out_rgb, stream)


def pic_decode_noalloc_check(stream=None) -> int:
    return load_library().pic_decode_noalloc_check(stream)


def pic_decode_test_wait_fault(withhold_arrival: int, spin_limit: int) -> int:
    return load_library().pic_decode_test_wait_fault(withhold_arrival, spin_limit)


def pic_decode_check(h, stream=None) -> int:
    return load_library().pic_decode_check(h, stream)


def pic_decode_destroy(h) -> None:
    load_library().pic_decode_destroy(h)


def pic_decode_kernel_name(h) -> str:
    return load_library().pic_decode_kernel_name(h).decode()


def pic_latent_count(H, W, L, C) -> int:
    return int(load_library().pic_latent_count(H, W, L, C))


def pic_param_count(arch: pic_arch) -> int:
    return int(load_library().pic_param_count(ctypes.byref(arch)))


def pic_status_string(status: int) -> str:
    return load_library().pic_status_string(status).decode()


def pic_izpr_workspace_bytes(n_symbols) -> int:
    return int(load_library().pic_izpr_workspace_bytes(n_symbols))


def pic_izpr_decode(symbols, n_symbols, eob, n_blocks, coeffs, offsets, workspace,
                    workspace_bytes, stream=None) -> int:
    return load_library().pic_izpr_decode(symbols, n_symbols, eob, n_blocks, coeffs, offsets,
                                          workspace, workspace_bytes, stream)


def pic_izpr_status(workspace, stream=None) -> int:
    return load_library().pic_izpr_status(workspace, stream)


def izpr_decode(symbols, eob: int, n_blocks: int, stream=None):
    """Inverse ZpR of a device int32 symbol tensor; returns (coeffs [n][64]
    int32 raster order, offsets [n] int64) as torch CUDA tensors.  Raises if
    the stream is malformed (this synchronises the stream)."""
    import torch
    dev = symbols.device
    n = symbols.numel()
    coeffs = torch.empty((max(n_blocks, 1), 64), dtype=torch.int32, device=dev)[:n_blocks]
    offsets = torch.empty(max(n_blocks, 1), dtype=torch.int64, device=dev)[:n_blocks]
    wb = pic_izpr_workspace_bytes(n)
    ws = torch.empty(wb, dtype=torch.uint8, device=dev)
    sp = _stream_ptr(stream)
    rc = pic_izpr_decode(symbols.data_ptr() if n else None, n, int(eob), n_blocks,
                         coeffs.data_ptr() if n_blocks else None,
                         offsets.data_ptr() if n_blocks else None, ws.data_ptr(), wb, sp)
    if rc != PIC_OK:
        raise PicError(rc, "pic_izpr_decode")
    rc = pic_izpr_status(ws.data_ptr(), sp)
    if rc != PIC_OK:
        raise PicError(rc, "pic_izpr_status")
    return coeffs, offsets


def pic_idct_block_count(H, W, L, C) -> int:
    return int(load_library().pic_idct_block_count(H, W, L, C))


def pic_idct_unpatchify(coeffs, steps, B, H, W, L, C, latents, stream=None) -> int:
    return load_library().pic_idct_unpatchify(coeffs, steps, B, H, W, L, C, latents, stream)


def idct_unpatchify(coeffs, steps, H, W, L, C, out=None, stream=None):
    """Inverse DCT stage on torch CUDA tensors: coeffs int32 [B][n_blocks][64]
    (or [n_blocks][64] for one image), steps fp32 [B][L]; returns fp32
    latents [B][pic_latent_count] (enqueued on the stream, not synchronised)."""
    import torch
    n_blk = pic_idct_block_count(H, W, L, C)
    B = coeffs.numel() // (64 * n_blk) if n_blk > 0 else 0
    if B < 1 or coeffs.numel() != B * 64 * n_blk or steps.numel() != B * L:
        raise ValueError("idct_unpatchify: tensor sizes do not match the shapes")
    if out is None:
        out = torch.empty((B, pic_latent_count(H, W, L, C)), dtype=torch.float32,
                          device=coeffs.device)
    rc = pic_idct_unpatchify(coeffs.data_ptr(), steps.data_ptr(), B, H, W, L, C, out.data_ptr(),
                             _stream_ptr(stream))
    if rc != PIC_OK:
        raise PicError(rc, "pic_idct_unpatchify")
    return out


def pic_fuse_modulation(arch: pic_arch, B, shared, mod, weights_out, stream=None) -> int:
    return load_library().pic_fuse_modulation(ctypes.byref(arch), B, shared, mod, weights_out,
                                              stream)


def fuse_modulation(arch: pic_arch, shared, mod, out=None, stream=None):
    """App. A fusion on torch CUDA tensors: shared fp32 [P], mod fp32
    [B][4][C'] (gamma, beta, mu, sigma); returns the per-image weight blobs
    [B][P] (fp32, or fp16 for the tensor-core arch), enqueued on the stream."""
    import torch
    B = mod.shape[0]
    P = pic_param_count(arch)
    dt = torch.float32 if arch.precision == PIC_PREC_FP32 else torch.float16
    if out is None:
        out = torch.empty((B, P), dtype=dt, device=mod.device)
    rc = pic_fuse_modulation(arch, B, shared.data_ptr(), mod.data_ptr(), out.data_ptr(),
                             _stream_ptr(stream))
    if rc != PIC_OK:
        raise PicError(rc, "pic_fuse_modulation")
    return out


def pic_huffman_workspace_bytes(n_words, B, p) -> int:
    return int(load_library().pic_huffman_workspace_bytes(n_words, B, p))


def pic_huffman_decode(words, n_words, word_off, n_bits, B, tab_value, tab_len, max_table, p,
                       sym_off, out, workspace, workspace_bytes, stream=None) -> int:
    return load_library().pic_huffman_decode(words, n_words, word_off, n_bits, B, tab_value, tab_len,
                                             max_table, p, sym_off, out, workspace,
                                             workspace_bytes, stream)


def pic_huffman_status(workspace, stream=None) -> int:
    return load_library().pic_huffman_status(workspace, stream)


def fma_peak_tflops(device=None, iters: int = 8192, reps: int = 5) -> float:
    """Measured FP32 FMA throughput of the device (include/pic_measure.h):
    8 CTAs of 256 threads per SM, 3 warm-up launches, then reps launches
    timed with CUDA events on the current stream."""
    import torch
    dev = torch.device("cuda", torch.cuda.current_device()) if device is None else torch.device(device)
    blocks = 8 * torch.cuda.get_device_properties(dev).multi_processor_count
    out = torch.empty(blocks, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)
    sp = ctypes.c_void_p(stream.cuda_stream)
    lib = load_library()
    for _ in range(3):
        rc = lib.pic_fma_peak_launch(out.data_ptr(), blocks, iters, sp)
        if rc != PIC_OK:
            raise PicError(rc, "pic_fma_peak_launch")
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(reps):
        lib.pic_fma_peak_launch(out.data_ptr(), blocks, iters, sp)
    e1.record(stream)
    e1.synchronize()
    return lib.pic_fma_peak_flops(blocks, iters) * reps / (e0.elapsed_time(e1) * 1e-3) / 1e12


def huffman_decode(words, word_off, n_bits, tab_value, tab_len, p, sym_off, stream=None,
                   check=True):
    """Decodes B Huffman streams given as torch CUDA tensors (uint32 words as
    int32, int64 word_off [B+1], n_bits [B], int32 tables [B][max_table],
    int64 sym_off [B+1]); returns the int32 symbols [sym_off[B]].  With
    check, synchronises and raises if a stream is malformed."""
    import torch
    B = n_bits.numel()
    n_words = words.numel()
    total = int(sym_off[-1].item())
    out = torch.empty(max(total, 1), dtype=torch.int32, device=words.device)[:total]
    wb = pic_huffman_workspace_bytes(n_words, B, p)
    if wb < 0:
        raise ValueError("huffman_decode: arguments out of range")
    ws = torch.empty(wb, dtype=torch.uint8, device=words.device)
    sp = _stream_ptr(stream)
    rc = pic_huffman_decode(words.data_ptr(), n_words, word_off.data_ptr(), n_bits.data_ptr(), B,
                            tab_value.data_ptr(), tab_len.data_ptr(), tab_value.shape[-1], p,
                            sym_off.data_ptr(), out.data_ptr() if total else ws.data_ptr(),
                            ws.data_ptr(), wb, sp)
    if rc != PIC_OK:
        raise PicError(rc, "pic_huffman_decode")
    if check:
        rc = pic_huffman_status(ws.data_ptr(), sp)
        if rc != PIC_OK:
            raise PicError(rc, "pic_huffman_status")
    return out


# ---- convenience wrapper over torch tensors --------------------------------
def decode_buffer_bytes(arch: pic_arch, B, H, W) -> dict:
    """Bytes each buffer of a B-image H x W decode must hold at least:
    latents B x pic_latent_count x 4, steps B x L x 4 (int32 latents only),
    weights B x pic_param_count x (2 for the tensor-core arch, else 4), out
    B x 3 x H x W x (1 for uint8 output, else 4).  Sizes the C ABI would
    refuse count as 0 (the call itself then reports the error)."""
    B_, H_, W_ = max(B, 0), max(H, 0), max(W, 0)
    n_lat = max(pic_latent_count(H, W, arch.num_levels, arch.channels_per_level), 0)
    n_par = max(pic_param_count(arch), 0)
    return {
        "latents": 4 * B_ * n_lat,
        "steps": 4 * B_ * arch.num_levels if arch.latent_format == PIC_LATENT_INT32 else 0,
        "weights": (4 if arch.precision == PIC_PREC_FP32 else 2) * B_ * n_par,
        "out": (1 if arch.output_format == PIC_OUT_U8_HWC else 4) * 3 * B_ * H_ * W_,
    }


def check_decode_buffers(need: dict, B, H, W, host=False, device=None, **bufs):
    """Raises ValueError unless every named buffer (latents, steps, weights,
    out: torch tensors, or numpy arrays on the host path) is contiguous,
    lives on the device (host=False; on CUDA device index ``device`` when
    that is given) or the host (host=True), and holds at least
    ``need[name]`` bytes.  A missing (None) buffer passes only where the call
    does not read it."""
    for name, a in bufs.items():
        if a is None:
            if name != "steps" or need[name] > 0:
                raise ValueError(f"{name}: required by this decoder")
            continue
        if isinstance(a, np.ndarray):
            nbytes, contig, on_gpu = a.nbytes, a.flags["C_CONTIGUOUS"], False
        else:
            nbytes, contig, on_gpu = a.numel() * a.element_size(), a.is_contiguous(), a.is_cuda
        if not contig:
            raise ValueError(f"{name}: must be contiguous")
        if on_gpu == host:
            raise ValueError(f"{name}: must be a {'host' if host else 'CUDA'} buffer")
        if on_gpu and device is not None and a.device.index != device:
            raise ValueError(f"{name}: on cuda:{a.device.index}, but the decoder was created "
                             f"on cuda:{device}")
        if nbytes < need[name]:
            raise ValueError(f"{name}: holds {nbytes} bytes; a {B}-image {H}x{W} call needs "
                             f"{need[name]}")


def _stream_ptr(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return getattr(stream, "cuda_stream", stream)


class Decoder:
    """One decoder handle.  Tensors passed to the decode methods must be
    contiguous CUDA tensors of the documented dtypes.  The C ABI receives bare
    pointers and cannot see a buffer's size, so these methods refuse, before
    anything is launched, a buffer that is smaller than the call reads or
    writes, not contiguous, or on the wrong side of the host/device split."""

    def __init__(self, L, C, dims, act="relu", precision="fp32", clamp=True, max_H=1,
                 max_W=1, max_batch=1, latent="int32", output="f32_chw", staging="auto"):
        self.arch = make_arch(L, C, dims, act, precision, clamp, max_H, max_W, max_batch, latent,
                              output, staging)
        self.latent = latent
        self.L, self.C, self.dims, self.precision = L, C, tuple(dims), precision
        self._need = {}
        self.handle = pic_decode_create(self.arch)
        import torch
        self.device = torch.cuda.current_device()  # the handle's device (current at create)

    @classmethod
    def for_workload(cls, wl, precision: str, clamp=True, max_batch=None, latent="int32",
                     output="f32_chw", staging="auto"):
        return cls(wl.L, wl.C, wl.dims, wl.act, precision, clamp, wl.H, wl.W,
                   max_batch or wl.B, latent, output, staging)

    @property
    def kernel_name(self) -> str:
        return pic_decode_kernel_name(self.handle)

    def close(self):
        if self.handle:
            pic_decode_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    @staticmethod
    def _check(rc, where):
        if rc != PIC_OK:
            raise PicError(rc, where)

    def buffer_bytes(self, B, H, W) -> dict:
        """``decode_buffer_bytes`` for this handle's arch (cached per shape)."""
        key = (B, H, W)
        need = self._need.get(key)
        if need is None:
            if len(self._need) >= 64:
                self._need.clear()
            need = self._need[key] = decode_buffer_bytes(self.arch, B, H, W)
        return need

    def check_buffers(self, B, H, W, host=False, **bufs):
        check_decode_buffers(self.buffer_bytes(B, H, W), B, H, W, host,
                             None if host else self.device, **bufs)

    def decode_batch(self, latents, steps, weights, H, W, out, stream=None, B=None, check=True):
        """Enqueues a batch decode; arguments are torch CUDA tensors.  With
        check=False the buffer checks are skipped (a few microseconds of
        host time per call): for loops that reuse buffers already checked."""
        if B is None:
            B = out.shape[0] if out.dim() == 4 else 1
        if check:
            self.check_buffers(B, H, W, latents=latents, steps=steps, weights=weights, out=out)
        sp = steps.data_ptr() if steps is not None else None
        rc = pic_decode_batch(self.handle, B, latents.data_ptr(), sp,
                              weights.data_ptr(), H, W, out.data_ptr(), _stream_ptr(stream))
        self._check(rc, "pic_decode_batch")
        return out

    def decode(self, latents, steps, weights, H, W, out, stream=None):
        """Enqueues a one-image decode; arguments are torch CUDA tensors."""
        self.check_buffers(1, H, W, latents=latents, steps=steps, weights=weights, out=out)
        sp = steps.data_ptr() if steps is not None else None
        rc = pic_decode(self.handle, latents.data_ptr(), sp, weights.data_ptr(),
                        H, W, out.data_ptr(), _stream_ptr(stream))
        self._check(rc, "pic_decode")
        return out

    def decode_batch_host(self, latents: np.ndarray, steps: np.ndarray, weights: np.ndarray,
                          H, W, out: np.ndarray, stream=None, B=None):
        """Host buffers in (numpy arrays or CPU tensors, preferably pinned),
        host RGB out; copies and decodes inside the call, pipelined over
        chunks of images."""
        if B is None:
            B = latents.shape[0] if latents.ndim == 2 else 1
        self.check_buffers(B, H, W, host=True, latents=latents, steps=steps, weights=weights,
                           out=out)

        def ptr(a):
            if a is None:
                return None
            return a.ctypes.data if isinstance(a, np.ndarray) else a.data_ptr()

        rc = pic_decode_batch_host(self.handle, B, ptr(latents), ptr(steps), ptr(weights), H, W,
                                   ptr(out), _stream_ptr(stream))
        self._check(rc, "pic_decode_batch_host")
        return out

    def check(self, stream=None):
        self._check(pic_decode_check(self.handle, _stream_ptr(stream)), "pic_decode_check")
