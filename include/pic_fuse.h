/*
 * pic_fuse.h -- C ABI of the modulation fusion (arxiv 2609.09020, Sec. 3.1,
 * Eqs. 2-3, and App. A): the synthesis g_s is MLP^s (every layer but the
 * last, shared by all images) followed by MLP^i (the last linear layer).
 * For one image the encoder normalises the MLP^s output features per channel
 * over the image's pixels, (f - mu) / sigma, and modulates them,
 * gamma (.) + beta.  App. A folds both into MLP^i, so the decoder only needs
 *     w'[i][c] = w[i][c] gamma_c / sigma_c,
 *     b'[i]    = b[i] + sum_c w[i][c] (beta_c - gamma_c mu_c / sigma_c).
 * This entry point writes the per-image weight blobs that pic_decode_batch
 * consumes from the shared weights and every image's (gamma, beta, mu, sigma).
 *
 * Conventions as in pic_decode.h: device pointers owned by the caller,
 * asynchronous on `stream`, pic_status codes, no traps.
 */
#ifndef PIC_FUSE_H
#define PIC_FUSE_H

#include "pic_decode.h"

#ifdef __cplusplus
extern "C" {
#endif

/*
 * For B images:
 *   arch        : the decoder's architecture (num_layers >= 2); its precision
 *                 selects the output dtype (fp32, or IEEE half rounded to
 *                 nearest for the tensor-core precisions)
 *   shared      : float, device, [pic_param_count(arch)] -- the g_s weights in
 *                 the layout of pic_decode.h
 *   mod         : float, device, [B][4][C'] with C' = dims[num_layers - 1]:
 *                 per image the rows gamma, beta, mu, sigma (sigma > 0)
 *   weights_out : device, [B][pic_param_count(arch)] in the output dtype,
 *                 16-byte aligned: every layer of `shared` copied, the last
 *                 layer replaced by (w', b')
 * Errors: PIC_ERR_INVALID_ARG (NULL or misaligned pointers, B < 1, an arch
 * with fewer than 2 layers or inconsistent dims) with nothing launched;
 * PIC_ERR_CUDA if the launch failed.
 */
int pic_fuse_modulation(const pic_arch *arch, int B, const float *shared, const float *mod,
                        void *weights_out, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* PIC_FUSE_H */
