/*
 * pic_measure.h -- C ABI of the measurement helpers that sit beside the
 * decoder: an FP32 FMA throughput microbenchmark, the peak against which the
 * fp32 CUDA-core decode path's roofline fraction is reported (the decode
 * itself does not use it).
 *
 * Conventions as in pic_decode.h: asynchronous on `stream`, status codes
 * (pic_status values), no traps.
 */
#ifndef PIC_MEASURE_H
#define PIC_MEASURE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Floating-point operations (2 per FMA) of one pic_fma_peak_launch with
 * these arguments, or -1 for blocks < 1 or iters < 1. */
int64_t pic_fma_peak_flops(int blocks, int iters);

/*
 * Launches `blocks` CTAs of 256 threads; every thread runs iters x 128
 * dependent-chain FMAs spread over 8 independent chains, on registers only.
 *   out    : float, device, [blocks]; written only in a case that does not
 *            occur (it keeps the arithmetic from being optimised away)
 *   blocks : >= 1 (a multiple of the SM count x 8 fills every SM)
 *   iters  : >= 1
 * Errors: PIC_ERR_INVALID_ARG (NULL out, blocks or iters < 1), PIC_ERR_CUDA
 * (launch failure).
 */
int pic_fma_peak_launch(float *out, int blocks, int iters, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* PIC_MEASURE_H */
