/*
 * pic_izpr.h -- C ABI of the GPU inverse ZpR (arxiv 2609.09020, Sec. 3.3 and
 * Fig. 2: zigzag reorder, trailing-zero trim and zero-only run-length coding
 * of quantised 8x8 DCT blocks; App. B, Algorithm 1: the decoder's expansion
 * of the symbol stream, one block per end-of-block marker, after the marker
 * offsets have been found by a stream compaction).
 *
 * Stream format (the reading of Fig. 2 used throughout): one end-of-block
 * value `eob` per stream, larger than every literal by at least 17.  The 16
 * values eob-16 .. eob-1 code runs of 1..16 zeros (eob - 17 + n codes n
 * zeros), smaller values are literal coefficients written in zigzag order,
 * eob ends a block, and positions after a block's last symbol are zero.
 *
 * Conventions as in pic_decode.h: device pointers owned by the caller,
 * asynchronous on `stream`, status codes (pic_status values), no traps.
 */
#ifndef PIC_IZPR_H
#define PIC_IZPR_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Bytes of device workspace pic_izpr_decode needs for n_symbols symbols (a
 * status word and the compaction's marker counts: per 2048-symbol chunk its
 * offset within its group of 8 chunks, per group its count and base), or -1
 * for n_symbols < 0. */
int64_t pic_izpr_workspace_bytes(int64_t n_symbols);

/*
 * Inverse ZpR on `stream`:
 *   symbols   : int32, device, [n_symbols] (n_symbols >= 0)
 *   eob       : the stream's end-of-block value
 *   n_blocks  : number of blocks (= number of eob markers), >= 0
 *   coeffs    : int32, device, [n_blocks][64], raster order (row * 8 + col);
 *               every element is written
 *   offsets   : int64, device, [n_blocks]; receives the stream index of each
 *               block's marker (Algorithm 1's offsets)
 *   workspace : device, >= pic_izpr_workspace_bytes(n_symbols) bytes,
 *               16-byte aligned, caller-owned; it must not be shared by
 *               decodes that overlap on the GPU
 * A malformed stream (a block covering more than 64 positions, a value above
 * eob, a marker count different from n_blocks, or symbols after the last
 * marker) is recorded in the
 * workspace and reported by pic_izpr_status; the coefficients of the blocks
 * concerned are then unspecified, but nothing is written out of bounds.
 * Errors: PIC_ERR_INVALID_ARG (NULL or misaligned pointers, negative sizes,
 * workspace too small), PIC_ERR_CUDA (launch failure).
 */
int pic_izpr_decode(const int32_t *symbols, int64_t n_symbols, int32_t eob, int64_t n_blocks,
                    int32_t *coeffs, int64_t *offsets, void *workspace, size_t workspace_bytes,
                    void *stream);

/* Synchronises `stream` and returns PIC_OK if the last pic_izpr_decode that
 * used `workspace` found the stream well formed, PIC_ERR_INVALID_ARG if it
 * did not (or workspace is NULL), PIC_ERR_CUDA on a CUDA failure. */
int pic_izpr_status(const void *workspace, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* PIC_IZPR_H */
