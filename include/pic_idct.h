/*
 * pic_idct.h -- C ABI of the GPU inverse DCT stage (arxiv 2609.09020, Fig. 1
 * and Sec. 3.2, Eqs. 5-7: the encoder cuts every latent plane into 8 x 8
 * patches (z = Patchify(y_1..y_L)) and codes their quantised DCT
 * coefficients (s = DCT(z)); the decoder dequantises the coefficients, takes
 * the inverse DCT of every patch and puts the patches back into the latent
 * pyramid that the synthesis g_r of pic_decode.h reads).
 *
 * Conventions (the readings the oracle shares):
 *   - DCT is the orthonormal 2-D DCT-II on 8 x 8 blocks; its inverse is
 *       x[m][n] = sum_u sum_v a(u) a(v) S[u][v] cos((2m+1) u pi / 16) cos((2n+1) v pi / 16),
 *     a(0) = sqrt(1/8), a(k > 0) = 1/2.  A block is row-major, coefficient
 *     (u, v) at u * 8 + v (the raster order pic_izpr_decode writes).
 *   - Patch order: level l = 0..L-1 (finest first), channel c, patch row by,
 *     patch column bx; a level has ceil(H_l / 8) x ceil(W_l / 8) patches per
 *     channel and the positions of a ragged patch past the plane's edge are
 *     dropped.
 *   - Dequantisation multiplies the coefficients of a level-l patch by the
 *     level's step (step 1 is the paper's unit quantisation step).
 * Device pointers owned by the caller, asynchronous on `stream`, pic_status
 * codes, no traps.
 */
#ifndef PIC_IDCT_H
#define PIC_IDCT_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Number of 8 x 8 patches of one pyramid, sum_l C ceil(H_l/8) ceil(W_l/8),
 * H_l = ceil(H / 2^l); -1 for sizes out of range (H, W >= 1, L in 1..12,
 * C in 1..4). */
int64_t pic_idct_block_count(int H, int W, int L, int C);

/*
 * Inverse DCT stage for B images of the same shape, on `stream`:
 *   coeffs  : int32, device, [B][pic_idct_block_count][64], 16-byte aligned
 *   steps   : float, device, [B][L]
 *   latents : float, device, [B][pic_latent_count(H, W, L, C)] in the
 *             pyramid layout of pic_decode.h; every element is written
 * Errors: PIC_ERR_INVALID_ARG (NULL or misaligned pointers, sizes out of
 * range) with nothing launched; PIC_ERR_CUDA if the launch failed.
 */
int pic_idct_unpatchify(const int32_t *coeffs, const float *steps, int B, int H, int W, int L,
                        int C, float *latents, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* PIC_IDCT_H */
