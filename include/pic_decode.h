/*
 * pic_decode.h -- C ABI of the GB300 decoder for the PIC synthesis g_r
 * (arxiv 2609.09020, "PIC: Revisiting INR for Image Coding with Fast Encoding
 * and Sub-Millisecond Decoding").
 *
 * The decode problem (Sec. 3.1, Eq. 1; Sec. 4.1; App. A): an H x W image is
 * represented by L quantised latent grids y_hat = {y_l}, level l of size
 * ceil(H / 2^l) x ceil(W / 2^l) with C channels (l = 0 is full resolution;
 * the paper's index is i = L - l), plus the weights of the per-pixel synthesis
 * MLP g_s (the decoder only needs the fused weights w', b' of App. A).  For
 * every output pixel the decoder
 *   1. dequantises the integer symbols of every level: y = q * step_l,
 *   2. upsamples every level to H x W (bilinear, half-pixel centres, edge
 *      clamp, source coordinate (x + 1/2) * W_l / W - 1/2),
 *   3. concatenates the levels into a feature of L * C values (level-major,
 *      finest level first, channel-minor),
 *   4. runs g_s: h_{k+1} = act(W_k h_k + b_k) for hidden layers (act = ReLU,
 *      or GELU in its erf form), a linear last layer with 3 outputs,
 *   5. clamps the RGB result to [0, 1].
 * Steps 1-5 run fused in one kernel launch per call: features and hidden
 * activations never leave the chip.
 *
 * Conventions for every entry point below:
 *   - Device pointers are CUDA global-memory pointers on the current device,
 *     owned by the caller, contiguous, at least 16-byte aligned; the library
 *     never takes ownership of, frees, or keeps them after the call.
 *   - `stream` is a cudaStream_t (NULL = the legacy default stream).  Decode
 *     calls are asynchronous on it: they enqueue work and return without a
 *     host synchronisation.  Outputs are ready when the stream reaches them.
 *   - Every function returns a pic_status.  Argument errors are detected on
 *     the host before anything is launched.  No function calls exit(),
 *     abort() or traps on the device.
 *   - A handle is not thread-safe: calls on one handle must not overlap in
 *     host threads.  Different handles are independent.
 */
#ifndef PIC_DECODE_H
#define PIC_DECODE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct pic_decoder pic_decoder; /* opaque handle */

typedef enum {
    PIC_OK = 0,
    PIC_ERR_INVALID_ARG = -1, /* NULL pointer, bad size, misaligned pointer, arch mismatch */
    PIC_ERR_UNSUPPORTED = -2, /* arch outside the supported envelope, or no sm_103 device */
    PIC_ERR_CUDA = -3,        /* a CUDA runtime call or kernel launch failed */
    PIC_ERR_ALLOC = -4,       /* device allocation failed (create; first host-buffer call) */
    PIC_ERR_TIMEOUT = -5      /* a bounded device-side wait gave up (reported by pic_decode_check) */
} pic_status;

typedef enum {
    PIC_ACT_RELU = 0, /* max(z, 0) (Sec. 4.1) */
    PIC_ACT_GELU = 1  /* z * Phi(z) = z/2 (1 + erf(z / sqrt 2)) */
} pic_act;

typedef enum {
    /* fp32 weights; all arithmetic in fp32 on the CUDA cores. */
    PIC_PREC_FP32 = 0,
    /* fp16 weights; the MLP runs on the tensor cores with fp16 operands and
     * fp32 accumulation.  Every activation operand (features and hidden
     * values) is split into two fp16 terms hi + lo, so the products carry
     * about 22 significant bits; the weights are used exactly as given. */
    PIC_PREC_FP16_TC = 1,
    /* fp16 weights; tensor cores as PIC_PREC_FP16_TC, with the lo term of
     * every hidden operand in fp8 (e4m3) against an e4m3 copy of the
     * weights, the hidden activations kept scaled by 2^6: about 15
     * significant bits per product and half the lo MMAs.  For ReLU nets with
     * a hidden width of 64 and the output layer on the tensor cores (the
     * 7-64-64-3 architecture); hidden activations must stay below 1024 in
     * magnitude. */
    PIC_PREC_FP16_TC_LO8 = 2
} pic_prec;

typedef enum {
    /* int32 latent symbols q; the decode dequantises them, y_l = q * step_l. */
    PIC_LATENT_INT32 = 0,
    /* fp32 real latents, already dequantised -- the output of the inverse DCT
     * stage of pic_idct.h (Fig. 1: iDCT then g_r).  `steps` is not read and
     * may be NULL. */
    PIC_LATENT_FP32 = 1
} pic_latent_format;

typedef enum {
    /* The library's choice per architecture (measured: TMA where it is as
     * fast as per-thread copies, per-thread copies where TMA was slower). */
    PIC_STAGING_AUTO = 0,
    /* Every latent word a tile needs is loaded by the decoding threads'
     * 4-byte asynchronous copies, one tile ahead. */
    PIC_STAGING_COPIES = 1,
    /* A tile's full-resolution row (every channel) arrives as TMA boxes
     * issued two tiles ahead; the coarser levels' rows stay with per-thread
     * copies.  Tensor-core path only, for the architectures that have a
     * TMA-staged kernel (PIC_ERR_UNSUPPORTED at create otherwise); a call
     * whose latent buffer holds 2^31 words or more falls back to copies. */
    PIC_STAGING_TMA = 2
} pic_staging;

typedef enum {
    PIC_OUT_F32_CHW = 0, /* fp32 planar [3][H][W] (R, G, B planes) -- the default */
    PIC_OUT_F32_HWC = 1, /* fp32 interleaved [H][W][3] */
    PIC_OUT_U8_HWC = 2   /* uint8 interleaved [H][W][3]: round-half-even(255 clamp(v, 0, 1)) */
} pic_output_format;

/* Architecture of one decoder instance (fixed at create). */
typedef struct {
    int num_levels;         /* L, 1..12 */
    int channels_per_level; /* C, 1..4 */
    int num_layers;         /* n linear layers, 1..6 */
    int dims[7];            /* dims[0] = L*C, dims[n] = 3; every dim 1..128 */
    int hidden_act;         /* pic_act */
    int precision;          /* pic_prec */
    int clamp_output;       /* 1: clamp to [0, 1] (the decode); 0: raw MLP output */
    int max_H, max_W;       /* largest image accepted by the decode calls */
    int max_batch;          /* largest B accepted by pic_decode_batch */
    int latent_format;      /* pic_latent_format; same layout and size (4 B) either way */
    int output_format;      /* pic_output_format (uint8 output always clamps) */
    int staging;            /* pic_staging: how the tensor-core kernel stages latents */
} pic_arch;

/*
 * Creates a decoder for `arch` on the current CUDA device.  Validates the
 * arch, selects the kernel, and allocates the handle's small device state.
 * May synchronise.  On success *out receives the handle (destroy it with
 * pic_decode_destroy); on failure *out is set to NULL.
 * Errors: PIC_ERR_INVALID_ARG (NULL arch/out, inconsistent dims),
 * PIC_ERR_UNSUPPORTED (limits above, or the current device is not sm_103),
 * PIC_ERR_ALLOC, PIC_ERR_CUDA.
 */
int pic_decode_create(const pic_arch *arch, pic_decoder **out);

/*
 * Decodes one image (steps 1-5 above) on `stream`.
 *   latents : device; levels l = 0..L-1 concatenated, each planar
 *             [C][H_l][W_l] row-major, H_l = ceil(H / 2^l), W_l = ceil(W / 2^l);
 *             pic_latent_count(H, W, L, C) values: int32 symbols, or fp32
 *             values (passed through the same pointer) when the arch's
 *             latent_format is PIC_LATENT_FP32.
 *   steps   : float, device; [L] dequantisation step of each level (not read,
 *             and may be NULL, for PIC_LATENT_FP32).
 *   weights : device; for k = 0..n-1: W_k [dims[k+1]][dims[k]] row-major, then
 *             b_k [dims[k+1]]; pic_param_count(arch) values; float for
 *             PIC_PREC_FP32, IEEE half (uint16 bits) for PIC_PREC_FP16_TC.
 *   H, W    : image size, 1..max_H, 1..max_W.
 *   out_rgb : device, 16-byte aligned, in the arch's output_format: fp32
 *             planar [3][H][W] (R, G, B planes), fp32 [H][W][3], or uint8
 *             [H][W][3].
 * Errors: PIC_ERR_INVALID_ARG (NULL handle/pointer, misaligned pointer, H or W
 * out of range, or the current device is not the one the handle was created
 * on) with nothing launched; PIC_ERR_CUDA if the launch failed.
 */
int pic_decode(pic_decoder *h, const int32_t *latents, const float *steps, const void *weights,
               int H, int W, void *out_rgb, void *stream);

/*
 * Decodes B independent images of the same size in one launch.  Image b uses
 * latents + b * pic_latent_count(H, W, L, C), steps + b * L,
 * weights + b * pic_param_count(arch) and writes the image's 3 * H * W
 * outputs at out_rgb + b * 3 * H * W elements
 * (all images' buffers are contiguous, image-major).  B in 1..max_batch;
 * other arguments and errors as pic_decode.
 */
int pic_decode_batch(pic_decoder *h, int B, const int32_t *latents, const float *steps,
                     const void *weights, int H, int W, void *out_rgb, void *stream);

/*
 * End-to-end convenience for callers holding HOST buffers (same layouts as
 * pic_decode_batch, host pointers): copies the inputs to device buffers owned
 * by the handle, decodes, copies the RGB back, and synchronises `stream`
 * before returning.  The batch runs as a pipeline over up to 16 chunks of
 * images on three internal streams (copy-in, decode, copy-out), ordered after
 * the work already queued on `stream`, so that the copies of one chunk
 * overlap the decode of another; the first two chunks are one and two images,
 * so that the copy-back starts early.  The output is identical to
 * pic_decode_batch's.  The copies overlap only when the host buffers are
 * page-locked (cudaHostAlloc / cudaHostRegister); with pageable memory the
 * result is the same but the copies run one after another.  The staging buffers and streams are allocated on
 * first use (for max_batch images of max_H x max_W) and kept until destroy;
 * calls on one handle must not overlap.
 * Errors: as pic_decode_batch, plus PIC_ERR_ALLOC.
 */
int pic_decode_batch_host(pic_decoder *h, int B, const int32_t *latents, const float *steps,
                          const void *weights, int H, int W, void *out_rgb, void *stream);

/*
 * Synchronises `stream` and reports whether any kernel of this handle
 * launched on it since the last check hit a bounded device-side wait limit
 * (PIC_ERR_TIMEOUT; the handle's flag is then cleared), or PIC_OK.
 * Errors: PIC_ERR_INVALID_ARG (NULL handle), PIC_ERR_CUDA.
 */
int pic_decode_check(pic_decoder *h, void *stream);

/*
 * Allocation-free decode (no counterpart in the paper).  For callers that
 * cannot call cudaMalloc: a plug-in whose host application hands out all
 * device memory from its own pool, a real-time loop that cannot accept
 * cudaMalloc's implicit device synchronisation and unbounded latency, a
 * service whose memory budget is fixed before it starts.
 * Same decode, layouts and argument rules as pic_decode_batch, with the
 * architecture passed directly instead of a handle (arch->max_H, max_W and
 * max_batch bound H, W and B as for a handle).  The caller passes inputs and
 * outputs; the call allocates nothing (no cudaMalloc, no cudaFree, no
 * allocating library routine).  The only global memory it uses besides the
 * caller's buffers is a 256-byte static device array built into the library,
 * which every GPU that loads the library holds until the process exits: one
 * status word of it per device (a call that would need more is refused).
 * The first call on a device, with that device current, looks up the
 * array's device address, the device's capabilities and the kernel's launch
 * attributes, and caches them; make that first call before any stream
 * capture.
 * The status word is zero when the library loads and is raised (never
 * cleared) by a call in which a bounded device-side wait gives up; it stays
 * raised until pic_decode_noalloc_check reads and clears it.  All calls on a
 * device share the word, so a raised word says that some call since the
 * last check gave up, not which one, and calls that overlap on the GPU
 * (different streams, no ordering between them) race with a concurrent
 * check's clear.
 * Errors: as pic_decode_batch (PIC_ERR_INVALID_ARG, PIC_ERR_UNSUPPORTED,
 * PIC_ERR_CUDA); nothing is launched on an argument error.
 */
int pic_decode_batch_noalloc(const pic_arch *arch, int B, const int32_t *latents,
                             const float *steps, const void *weights, int H, int W,
                             void *out_rgb, void *stream);

/*
 * Status of the allocation-free calls on the current device (no counterpart
 * in the paper): synchronises `stream`, then returns PIC_ERR_TIMEOUT if a
 * bounded device-side wait gave up in any pic_decode_batch_noalloc call on
 * this device since the last check (and clears the word, on `stream`), else
 * PIC_OK.  Allocates nothing.
 * Errors: PIC_ERR_CUDA.
 */
int pic_decode_noalloc_check(void *stream);

/*
 * Test hook of the bounded device-side waits (no counterpart in the paper;
 * production code never calls it).  Every tensor-core decode launched while
 * withhold_arrival = 1 has one decoding thread of its first CTA skip one
 * mbarrier arrival, so that a wait of that CTA runs out and the kernel takes
 * its abort path (status word raised, remaining work skipped, outstanding
 * MMAs and copies drained, tensor memory freed); spin_limit > 0 replaces the
 * number of polls a wait makes before giving up (seconds' worth by default),
 * so that the wait runs out in microseconds.  pic_decode_test_wait_fault(0,
 * 0) restores production behaviour.  Process-wide, for all handles and the
 * allocation-free entry point; not synchronised with decode calls in other
 * host threads.
 * Errors: PIC_ERR_INVALID_ARG (withhold_arrival not 0 or 1).
 */
int pic_decode_test_wait_fault(int withhold_arrival, unsigned spin_limit);

/* Frees the handle and its device state.  NULL is a no-op.  Synchronises the
 * device first, so that no kernel of this handle is still running. */
void pic_decode_destroy(pic_decoder *h);

/* Name of the kernel the handle launches (static string), or "" for NULL:
 * the TMA-staged kernel where the handle stages with TMA (a call whose
 * latent buffer holds 2^31 words or more runs its per-thread-copy twin). */
const char *pic_decode_kernel_name(const pic_decoder *h);

/* sum_l C * ceil(H/2^l) * ceil(W/2^l), or -1 for invalid arguments. */
int64_t pic_latent_count(int H, int W, int L, int C);

/* sum_k dims[k+1] * (dims[k] + 1), or -1 for an invalid arch. */
int64_t pic_param_count(const pic_arch *arch);

/* Static description of a status code. */
const char *pic_status_string(int status);

#ifdef __cplusplus
}
#endif

#endif /* PIC_DECODE_H */
