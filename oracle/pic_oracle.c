/*
 * pic_oracle.c -- plain, slow, fp64 CPU decoder for the PIC synthesis g_r
 * (Sec. 3.1, Eq. 1; Sec. 3.3; Sec. 4.1 "Implementation Details"; App. A).
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the parity oracle for the CUDA
 * decoder.  Only the test suite, the smoke check and the CPU-baseline leg of
 * the benchmark load it.  It shares no code, header, table or constant with
 * the CUDA path, and the CUDA path never calls it.
 *
 * What it computes, per output pixel (x, y) of an H x W image:
 *   1. dequantisation of the integer latent symbols of every pyramid level
 *      (Fig. 1: the decoder reconstructs real latents from quantised symbols):
 *          y_l[c][v][u] = q_l[c][v][u] * step_l
 *   2. upsampling of every level to H x W (Sec. 3.1, after Eq. 1: the levels
 *      of y_hat are brought to one grid, y_u in R^{C x H x W}).  The paper does not name the
 *      kernel; this oracle uses bilinear interpolation with half-pixel
 *      centres and edge clamping, the size-based scale W_l / W and H_l / H.
 *   3. per-pixel concatenation of all levels into the feature vector that
 *      feeds g_s (Sec. 3.1: y_u has C channels at every pixel).  Order:
 *      level-major, finest level first, channel-minor.
 *   4. the synthesis MLP g_s (Sec. 4.1: an MLP with ReLU activations; the
 *      decoder only needs the fused weights w', b', App. A):
 *          h_{k+1} = act(W_k h_k + b_k) for hidden layers, linear last layer.
 *      act is ReLU, or GELU in its exact erf form.
 *   5. clamp of the RGB output to [0, 1].
 *
 * Notation: the paper numbers levels i = 1..L with i = L the finest
 * (H_i = H / 2^(L-i), Eq. 1).  Here l = L - i, so l = 0 is the full-resolution
 * level and H_l = ceil(H / 2^l), W_l = ceil(W / 2^l) (Eq. 1 assumes exact
 * division; the ceiling covers sizes that are not multiples of 2^l).
 *
 * Memory layouts (all row-major, contiguous):
 *   latents : levels l = 0..L-1 concatenated, each level planar [C][H_l][W_l]
 *   steps   : [L]
 *   weights : for k = 0..n-1: W_k [dims[k+1]][dims[k]] then b_k [dims[k+1]]
 *   out_rgb : planar [3][H][W]
 *
 * Arithmetic is double throughout, every sum in index order; build with
 * -O2 -ffp-contract=off so that no fused multiply-add changes the rounding.
 */
#include <math.h>
#include <stdint.h>
#include <stddef.h>

#define PIC_ORACLE_ACT_RELU 0
#define PIC_ORACLE_ACT_GELU 1

#define PIC_ORACLE_MAX_LEVELS 16
#define PIC_ORACLE_MAX_WIDTH 512

/* Size of pyramid level l: ceil(n / 2^l) (Eq. 1, ceiling reading). */
static int level_size(int n, int l)
{
    int64_t p = (int64_t)1 << l;
    return (int)(((int64_t)n + p - 1) / p);
}

int pic_oracle_level_size(int n, int l)
{
    if (n <= 0 || l < 0 || l > 30) return -1;
    return level_size(n, l);
}

/* Number of int32 symbols of one image's pyramid: sum_l C * H_l * W_l. */
int64_t pic_oracle_latent_count(int H, int W, int L, int C)
{
    int64_t n = 0;
    for (int l = 0; l < L; ++l)
        n += (int64_t)C * level_size(H, l) * level_size(W, l);
    return n;
}

/* Number of weight + bias values of the MLP: sum_k d_{k+1} (d_k + 1). */
int64_t pic_oracle_param_count(int n_layers, const int *dims)
{
    int64_t n = 0;
    for (int k = 0; k < n_layers; ++k)
        n += (int64_t)dims[k + 1] * dims[k] + dims[k + 1];
    return n;
}

/* Step 1: dequantisation y = q * step, element by element. */
void pic_oracle_dequant(const int32_t *q, int64_t n, double step, double *y)
{
    for (int64_t i = 0; i < n; ++i)
        y[i] = (double)q[i] * step;
}

/*
 * Step 2 at one output pixel: bilinear sample of a Hl x Wl grid g, seen as an
 * image stretched over H x W output pixels.  The source coordinate of output
 * pixel centre x + 1/2 is (x + 1/2) * Wl / W - 1/2, clamped below at 0; the
 * right/bottom neighbour index is clamped at the last row/column.
 */
double pic_oracle_bilinear_at(const double *g, int Hl, int Wl, int H, int W,
                              int x, int y)
{
    double sx = ((double)x + 0.5) * ((double)Wl / (double)W) - 0.5;
    double sy = ((double)y + 0.5) * ((double)Hl / (double)H) - 0.5;
    if (sx < 0.0) sx = 0.0;
    if (sy < 0.0) sy = 0.0;
    int u0 = (int)floor(sx);
    int v0 = (int)floor(sy);
    int u1 = (u0 + 1 < Wl) ? u0 + 1 : Wl - 1;
    int v1 = (v0 + 1 < Hl) ? v0 + 1 : Hl - 1;
    double a = sx - (double)u0; /* weight of column u1 */
    double b = sy - (double)v0; /* weight of row v1 */
    double top = (1.0 - a) * g[(int64_t)v0 * Wl + u0] + a * g[(int64_t)v0 * Wl + u1];
    double bot = (1.0 - a) * g[(int64_t)v1 * Wl + u0] + a * g[(int64_t)v1 * Wl + u1];
    return (1.0 - b) * top + b * bot;
}

/* Step 2 over a whole image: out[y][x] = bilinear sample at (x, y). */
void pic_oracle_upsample(const double *g, int Hl, int Wl, int H, int W, double *out)
{
    for (int y = 0; y < H; ++y)
        for (int x = 0; x < W; ++x)
            out[(int64_t)y * W + x] = pic_oracle_bilinear_at(g, Hl, Wl, H, W, x, y);
}

/* Hidden activation.  GELU(z) = z * Phi(z) = 0.5 z (1 + erf(z / sqrt 2)). */
double pic_oracle_act(double z, int act)
{
    if (act == PIC_ORACLE_ACT_GELU)
        return 0.5 * z * (1.0 + erf(z / sqrt(2.0)));
    return z > 0.0 ? z : 0.0;
}

/*
 * Step 4: g_s on one feature vector.  W_k is [dims[k+1]][dims[k]] row-major
 * followed by b_k; z_i = sum_j W_k[i][j] h_j + b_k[i], summed in j order.
 * Returns 0, or -1 for unsupported dims.
 */
int pic_oracle_mlp(const double *in, const double *weights, int n_layers,
                   const int *dims, int act, double *out)
{
    double h[PIC_ORACLE_MAX_WIDTH], z[PIC_ORACLE_MAX_WIDTH];
    if (n_layers < 1) return -1;
    for (int k = 0; k <= n_layers; ++k)
        if (dims[k] < 1 || dims[k] > PIC_ORACLE_MAX_WIDTH) return -1;
    for (int j = 0; j < dims[0]; ++j) h[j] = in[j];
    const double *p = weights;
    for (int k = 0; k < n_layers; ++k) {
        int din = dims[k], dout = dims[k + 1];
        const double *Wk = p;
        const double *bk = p + (int64_t)dout * din;
        for (int i = 0; i < dout; ++i) {
            double s = 0.0;
            for (int j = 0; j < din; ++j) s += Wk[(int64_t)i * din + j] * h[j];
            z[i] = s + bk[i];
        }
        int last = (k == n_layers - 1);
        for (int i = 0; i < dout; ++i) h[i] = last ? z[i] : pic_oracle_act(z[i], act);
        p = bk + dout;
    }
    for (int i = 0; i < dims[n_layers]; ++i) out[i] = h[i];
    return 0;
}

/* Step 5: clamp to [0, 1]. */
double pic_oracle_clamp01(double v)
{
    if (v < 0.0) return 0.0;
    if (v > 1.0) return 1.0;
    return v;
}

/* The 8-bit output variant: round-half-even(255 clamp(v, 0, 1)) (the decode
 * statement's clamp to [0, 1], scaled to the byte range). */
int pic_oracle_to_u8(double v)
{
    return (int)nearbyint(255.0 * pic_oracle_clamp01(v));
}

/* Checks shared by the two decode entry points. */
static int check_args(int H, int W, int L, int C, int n_layers, const int *dims)
{
    if (H < 1 || W < 1 || L < 1 || L > PIC_ORACLE_MAX_LEVELS || C < 1) return -1;
    if (n_layers < 1 || dims[0] != L * C || dims[n_layers] != 3) return -1;
    for (int k = 0; k <= n_layers; ++k)
        if (dims[k] < 1 || dims[k] > PIC_ORACLE_MAX_WIDTH) return -1;
    return 0;
}

/* The upsampled feature vector of pixel (x, yy) (steps 2-3). */
static void features_at(double *const *y, int L, int C, int H, int W, int x, int yy, double *f)
{
    int d = 0;
    for (int l = 0; l < L; ++l) {
        int Hl = level_size(H, l), Wl = level_size(W, l);
        for (int c = 0; c < C; ++c)
            f[d++] = pic_oracle_bilinear_at(y[l] + (int64_t)c * Hl * Wl, Hl, Wl, H, W, x, yy);
    }
}

/*
 * Steps 1-5 at one pixel, given the dequantised levels y[l] (planar [C][H_l][W_l]).
 */
static int decode_pixel(double *const *y, int L, int C, const double *weights,
                        int n_layers, const int *dims, int act, int clamp,
                        int H, int W, int x, int yy, double *rgb)
{
    double f[PIC_ORACLE_MAX_WIDTH];
    features_at(y, L, C, H, W, x, yy, f);
    if (pic_oracle_mlp(f, weights, n_layers, dims, act, rgb) != 0) return -1;
    if (clamp)
        for (int c = 0; c < 3; ++c) rgb[c] = pic_oracle_clamp01(rgb[c]);
    return 0;
}

/* Dequantises every level of one pyramid into `work`; fills y[l]. */
static void dequant_pyramid(const int32_t *latents, const double *steps, int L, int C,
                            int H, int W, double *work, double **y)
{
    int64_t off = 0;
    for (int l = 0; l < L; ++l) {
        int64_t n = (int64_t)C * level_size(H, l) * level_size(W, l);
        y[l] = work + off;
        pic_oracle_dequant(latents + off, n, steps[l], y[l]);
        off += n;
    }
}

/* Points y[l] at the levels of a pyramid of real values (no dequantisation). */
static void split_pyramid(const double *values, int L, int C, int H, int W, double **y)
{
    int64_t off = 0;
    for (int l = 0; l < L; ++l) {
        y[l] = (double *)(values + off);
        off += (int64_t)C * level_size(H, l) * level_size(W, l);
    }
}

/* Steps 2-5 over every pixel of one image, given its real-valued levels y[l]. */
static int decode_levels(double *const *y, const double *weights, int L, int C, int n_layers,
                         const int *dims, int act, int clamp, int H, int W, double *out_rgb,
                         int nthreads)
{
    int64_t plane = (int64_t)H * W;
    int bad = 0;
#ifdef _OPENMP
#pragma omp parallel for num_threads(nthreads > 0 ? nthreads : 1) schedule(static) reduction(| : bad)
#endif
    for (int yy = 0; yy < H; ++yy) {
        for (int x = 0; x < W; ++x) {
            double rgb[3];
            if (decode_pixel(y, L, C, weights, n_layers, dims, act, clamp, H, W, x, yy, rgb) != 0) {
                bad = 1;
                continue;
            }
            for (int c = 0; c < 3; ++c) out_rgb[c * plane + (int64_t)yy * W + x] = rgb[c];
        }
    }
    (void)nthreads;
    return bad ? -1 : 0;
}

/*
 * Full decode of one image.  `work` must hold pic_oracle_latent_count(H, W, L, C)
 * doubles.  nthreads > 1 splits the output rows over OpenMP threads (the
 * arithmetic of each pixel does not change).  Returns 0 or -1.
 */
int pic_oracle_decode(const int32_t *latents, const double *steps, const double *weights,
                      int L, int C, int n_layers, const int *dims, int act, int clamp,
                      int H, int W, double *out_rgb, double *work, int nthreads)
{
    double *y[PIC_ORACLE_MAX_LEVELS];
    if (check_args(H, W, L, C, n_layers, dims) != 0) return -1;
    dequant_pyramid(latents, steps, L, C, H, W, work, y);
    return decode_levels(y, weights, L, C, n_layers, dims, act, clamp, H, W, out_rgb, nthreads);
}

/*
 * Steps 2-5 of one image whose latents are already real values (the output
 * of the iDCT stage below, Fig. 1: iDCT then g_r), same layout as the
 * symbols of pic_oracle_decode.  Returns 0 or -1.
 */
int pic_oracle_decode_values(const double *latents, const double *weights, int L, int C,
                             int n_layers, const int *dims, int act, int clamp, int H, int W,
                             double *out_rgb, int nthreads)
{
    double *y[PIC_ORACLE_MAX_LEVELS];
    if (check_args(H, W, L, C, n_layers, dims) != 0) return -1;
    split_pyramid(latents, L, C, H, W, y);
    return decode_levels(y, weights, L, C, n_layers, dims, act, clamp, H, W, out_rgb, nthreads);
}

/*
 * Decode only the listed pixels (index y * W + x) of one image; out is
 * [npix][3].  Used to check full-size outputs at sampled positions.
 */
int pic_oracle_decode_pixels(const int32_t *latents, const double *steps, const double *weights,
                             int L, int C, int n_layers, const int *dims, int act, int clamp,
                             int H, int W, const int64_t *pix, int64_t npix, double *out,
                             double *work)
{
    double *y[PIC_ORACLE_MAX_LEVELS];
    if (check_args(H, W, L, C, n_layers, dims) != 0) return -1;
    dequant_pyramid(latents, steps, L, C, H, W, work, y);
    for (int64_t i = 0; i < npix; ++i) {
        if (pix[i] < 0 || pix[i] >= (int64_t)H * W) return -1;
        int yy = (int)(pix[i] / W), x = (int)(pix[i] % W);
        if (decode_pixel(y, L, C, weights, n_layers, dims, act, clamp, H, W, x, yy, out + 3 * i) != 0)
            return -1;
    }
    return 0;
}

/* ------------------------------------------------------------------------
 * ZpR and its inverse (Sec. 3.3, Fig. 2; App. B, Algorithm 1).
 *
 * A block is 8 x 8 quantised DCT coefficients, row-major (raster order).
 * ZpR reorders a block in zigzag order, trims its trailing zeros and codes
 * every run of zeros by its length (a partial run-length code: only zeros
 * are run-coded).
 * The stream uses one end-of-block marker value eob, larger than every
 * literal by at least 17: the 16 values eob-16 .. eob-1 code runs of 1..16
 * zeros (code eob - 17 + n for a run of n), any smaller value is a literal
 * coefficient, and eob itself ends a block.  Longer runs take several codes.
 * ------------------------------------------------------------------------ */

/* Zigzag order of an 8 x 8 block: order[k] is the raster index (row*8+col)
 * of the k-th coefficient.  Anti-diagonal d = row + col is walked with the
 * row falling for even d and rising for odd d, starting at (0, 0). */
void pic_oracle_zigzag(int *order)
{
    int k = 0;
    for (int d = 0; d <= 14; ++d) {
        int lo = d < 8 ? 0 : d - 7, hi = d < 8 ? d : 7;
        if (d % 2 == 0)
            for (int row = hi; row >= lo; --row) order[k++] = row * 8 + (d - row);
        else
            for (int row = lo; row <= hi; ++row) order[k++] = row * 8 + (d - row);
    }
}

/* Forward ZpR of n blocks (raster order) into symbols; returns the number of
 * symbols written, or -1 if cap is too small or a literal collides with the
 * run codes (coefficients must be < eob - 16). */
int64_t pic_oracle_zpr_encode(const int32_t *coeffs, int64_t n_blocks, int32_t eob,
                              int32_t *symbols, int64_t cap)
{
    int order[64];
    pic_oracle_zigzag(order);
    int64_t n = 0;
    for (int64_t b = 0; b < n_blocks; ++b) {
        const int32_t *blk = coeffs + 64 * b;
        int zz[64];
        for (int k = 0; k < 64; ++k) zz[k] = blk[order[k]];
        int last = -1; /* trim trailing zeros */
        for (int k = 0; k < 64; ++k)
            if (zz[k] != 0) last = k;
        int k = 0;
        while (k <= last) {
            if (zz[k] != 0) {
                if (zz[k] >= eob - 16) return -1;
                if (n >= cap) return -1;
                symbols[n++] = zz[k++];
            } else {
                int run = 0;
                while (k <= last && zz[k] == 0 && run < 16) { ++run; ++k; }
                if (n >= cap) return -1;
                symbols[n++] = eob - 17 + run;
            }
        }
        if (n >= cap) return -1;
        symbols[n++] = eob;
    }
    return n;
}

/* Inverse ZpR (Algorithm 1's expansion, done block after block): split the
 * stream at the eob markers, write literals and zero runs at consecutive
 * zigzag positions of the block, leave the trimmed tail zero.  Returns 0,
 * or -1 for a malformed stream (a block overflowing 64 positions, a
 * symbol >= eob other than the marker, or a marker count != n_blocks). */
int pic_oracle_izpr(const int32_t *symbols, int64_t n_symbols, int32_t eob,
                    int32_t *coeffs, int64_t n_blocks)
{
    int order[64];
    pic_oracle_zigzag(order);
    for (int64_t i = 0; i < 64 * n_blocks; ++i) coeffs[i] = 0;
    int64_t b = 0, pos = 0;
    for (int64_t i = 0; i < n_symbols; ++i) {
        int32_t s = symbols[i];
        if (s == eob) {
            ++b;
            pos = 0;
            continue;
        }
        if (b >= n_blocks || s > eob) return -1;
        int32_t *blk = coeffs + 64 * b;
        if (s >= eob - 16) {
            int run = s + 17 - eob;
            if (pos + run > 64) return -1;
            for (int r = 0; r < run; ++r) blk[order[pos++]] = 0;
        } else {
            if (pos + 1 > 64) return -1;
            blk[order[pos++]] = s;
        }
    }
    return b == n_blocks ? 0 : -1;
}

/* ------------------------------------------------------------------------
 * Patchify + DCT and their inverses (Fig. 1; Sec. 3.2, Eqs. 5-7).
 *
 * The encoder cuts every latent plane into 8 x 8 patches, concatenates them
 * (z = Patchify(y), Eq. 6) and takes their DCT (s = DCT(z), Eq. 7); the
 * quantised DCT coefficients are what ZpR codes.  The decoder runs the
 * inverse: dequantise the coefficients, inverse DCT, put every patch back.
 *
 * Readings (the paper names the steps only):
 *  - DCT is the orthonormal 2-D DCT-II of JPEG's transform,
 *        S[u][v] = a(u) a(v) sum_m sum_n x[m][n] cos((2m+1) u pi / 16) cos((2n+1) v pi / 16)
 *    with a(0) = sqrt(1/8), a(k > 0) = sqrt(2/8); its inverse (DCT-III) is
 *        x[m][n] = sum_u sum_v a(u) a(v) S[u][v] cos((2m+1) u pi / 16) cos((2n+1) v pi / 16).
 *    u, m index rows (vertical), v, n columns; a block is stored row-major,
 *    coefficient (u, v) at u * 8 + v, the raster order iZpR produces.
 *  - Patch order: levels l = 0..L-1 (finest first), then channel c, then
 *    patch row by, then patch column bx.  A plane whose side is not a
 *    multiple of 8 gets ceil(H_l / 8) x ceil(W_l / 8) patches; the encoder
 *    fills positions past the edge with the nearest edge value and the
 *    decoder drops them.
 *  - Dequantisation multiplies every coefficient of a level-l patch by the
 *    level's step (step = 1 is the paper's unit quantisation step).
 * ------------------------------------------------------------------------ */

static const double PIC_ORACLE_PI = 3.14159265358979323846;

static double dct_alpha(int k)
{
    return k == 0 ? sqrt(1.0 / 8.0) : sqrt(2.0 / 8.0);
}

/* Forward orthonormal 8x8 DCT-II of x (row-major) into S (row-major). */
void pic_oracle_dct8x8(const double *x, double *S)
{
    for (int u = 0; u < 8; ++u)
        for (int v = 0; v < 8; ++v) {
            double s = 0.0;
            for (int m = 0; m < 8; ++m)
                for (int n = 0; n < 8; ++n)
                    s += x[m * 8 + n] * cos((2 * m + 1) * u * PIC_ORACLE_PI / 16.0) *
                         cos((2 * n + 1) * v * PIC_ORACLE_PI / 16.0);
            S[u * 8 + v] = dct_alpha(u) * dct_alpha(v) * s;
        }
}

/* Inverse orthonormal 8x8 DCT (DCT-III) of S into x, both row-major. */
void pic_oracle_idct8x8(const double *S, double *x)
{
    for (int m = 0; m < 8; ++m)
        for (int n = 0; n < 8; ++n) {
            double s = 0.0;
            for (int u = 0; u < 8; ++u)
                for (int v = 0; v < 8; ++v)
                    s += dct_alpha(u) * dct_alpha(v) * S[u * 8 + v] *
                         cos((2 * m + 1) * u * PIC_ORACLE_PI / 16.0) *
                         cos((2 * n + 1) * v * PIC_ORACLE_PI / 16.0);
            x[m * 8 + n] = s;
        }
}

/* Number of 8x8 patches of one pyramid: sum_l C ceil(H_l / 8) ceil(W_l / 8). */
int64_t pic_oracle_block_count(int H, int W, int L, int C)
{
    int64_t n = 0;
    for (int l = 0; l < L; ++l)
        n += (int64_t)C * ((level_size(H, l) + 7) / 8) * ((level_size(W, l) + 7) / 8);
    return n;
}

/* Encoder side (for tests): Patchify (Eq. 6) then DCT (Eq. 7) of one
 * pyramid of real latents into coeffs [block_count][64].  Returns 0 or -1. */
int pic_oracle_patchify_dct(const double *latents, int H, int W, int L, int C, double *coeffs)
{
    if (H < 1 || W < 1 || L < 1 || L > PIC_ORACLE_MAX_LEVELS || C < 1) return -1;
    int64_t off = 0, b = 0;
    for (int l = 0; l < L; ++l) {
        int Hl = level_size(H, l), Wl = level_size(W, l);
        for (int c = 0; c < C; ++c) {
            const double *g = latents + off + (int64_t)c * Hl * Wl;
            for (int by = 0; by < (Hl + 7) / 8; ++by)
                for (int bx = 0; bx < (Wl + 7) / 8; ++bx, ++b) {
                    double x[64];
                    for (int m = 0; m < 8; ++m)
                        for (int n = 0; n < 8; ++n) {
                            int r = 8 * by + m, q = 8 * bx + n;
                            if (r > Hl - 1) r = Hl - 1;
                            if (q > Wl - 1) q = Wl - 1;
                            x[m * 8 + n] = g[(int64_t)r * Wl + q];
                        }
                    pic_oracle_dct8x8(x, coeffs + 64 * b);
                }
        }
        off += (int64_t)C * Hl * Wl;
    }
    return 0;
}

/* Decoder side: dequantise the integer coefficients of every patch by its
 * level's step, inverse DCT, and write the patch back into its plane,
 * dropping the positions past the plane's edge.  symbols is
 * [block_count][64], latents receives pic_oracle_latent_count values in the
 * pyramid layout.  Returns 0 or -1. */
int pic_oracle_unpatchify_idct(const int32_t *symbols, const double *steps, int H, int W, int L,
                               int C, double *latents)
{
    if (H < 1 || W < 1 || L < 1 || L > PIC_ORACLE_MAX_LEVELS || C < 1) return -1;
    int64_t off = 0, b = 0;
    for (int l = 0; l < L; ++l) {
        int Hl = level_size(H, l), Wl = level_size(W, l);
        for (int c = 0; c < C; ++c) {
            double *g = latents + off + (int64_t)c * Hl * Wl;
            for (int by = 0; by < (Hl + 7) / 8; ++by)
                for (int bx = 0; bx < (Wl + 7) / 8; ++bx, ++b) {
                    double S[64], x[64];
                    for (int k = 0; k < 64; ++k) S[k] = (double)symbols[64 * b + k] * steps[l];
                    pic_oracle_idct8x8(S, x);
                    for (int m = 0; m < 8; ++m)
                        for (int n = 0; n < 8; ++n) {
                            int r = 8 * by + m, q = 8 * bx + n;
                            if (r < Hl && q < Wl) g[(int64_t)r * Wl + q] = x[m * 8 + n];
                        }
                }
        }
        off += (int64_t)C * Hl * Wl;
    }
    return 0;
}

/* ------------------------------------------------------------------------
 * Modulation fusion (Sec. 3.1, Eqs. 2-3; App. A).
 *
 * g_s is MLP^s (every layer but the last, with its activations; shared by all
 * images) followed by MLP^i (the last, linear layer).  For one image the
 * encoder normalises the MLP^s output features f per channel over the H x W
 * pixels, fbar = (f - mu) / sigma, modulates them, ftilde = gamma fbar +
 * beta, and feeds ftilde to MLP^i.  App. A folds normalisation and
 * modulation into MLP^i's weights, so the decoder needs only
 *     w'[i][c] = w[i][c] gamma_c / sigma_c,
 *     b'[i]    = b[i] + sum_c w[i][c] (beta_c - gamma_c mu_c / sigma_c).
 * Reading: mean(f) and std(f) are the population mean and standard deviation
 * over the image's pixels (divide by N, no epsilon).
 * ------------------------------------------------------------------------ */

/* Per-channel population mean and standard deviation of f [C][N] (two passes). */
void pic_oracle_channel_stats(const double *f, int C, int64_t N, double *mu, double *sigma)
{
    for (int c = 0; c < C; ++c) {
        const double *x = f + (int64_t)c * N;
        double s = 0.0;
        for (int64_t i = 0; i < N; ++i) s += x[i];
        double m = s / (double)N, v = 0.0;
        for (int64_t i = 0; i < N; ++i) v += (x[i] - m) * (x[i] - m);
        mu[c] = m;
        sigma[c] = sqrt(v / (double)N);
    }
}

/* ftilde = gamma (f - mu) / sigma + beta, per channel, f and out [C][N]. */
void pic_oracle_norm_modulate(const double *f, int C, int64_t N, const double *mu,
                              const double *sigma, const double *gamma, const double *beta,
                              double *out)
{
    for (int c = 0; c < C; ++c)
        for (int64_t i = 0; i < N; ++i)
            out[(int64_t)c * N + i] =
                gamma[c] * ((f[(int64_t)c * N + i] - mu[c]) / sigma[c]) + beta[c];
}

/* App. A: the fused MLP^i layer w' [dout][C], b' [dout] from w, b, gamma, beta, mu, sigma. */
void pic_oracle_fuse_modulation(const double *w, const double *b, int dout, int C,
                                const double *gamma, const double *beta, const double *mu,
                                const double *sigma, double *w_out, double *b_out)
{
    for (int i = 0; i < dout; ++i) {
        double s = b[i];
        for (int c = 0; c < C; ++c) {
            w_out[(int64_t)i * C + c] = w[(int64_t)i * C + c] * gamma[c] / sigma[c];
            s += w[(int64_t)i * C + c] * (beta[c] - gamma[c] * mu[c] / sigma[c]);
        }
        b_out[i] = s;
    }
}

/* MLP^s at one pixel: the first n_layers - 1 layers, each followed by act;
 * f receives dims[n_layers - 1] values. */
static void mlps_at(const double *in, const double *weights, int n_layers, const int *dims,
                    int act, double *f)
{
    double h[PIC_ORACLE_MAX_WIDTH], z[PIC_ORACLE_MAX_WIDTH];
    for (int j = 0; j < dims[0]; ++j) h[j] = in[j];
    const double *p = weights;
    for (int k = 0; k < n_layers - 1; ++k) {
        int din = dims[k], dout = dims[k + 1];
        const double *Wk = p, *bk = p + (int64_t)dout * din;
        for (int i = 0; i < dout; ++i) {
            double acc = 0.0;
            for (int j = 0; j < din; ++j) acc += Wk[(int64_t)i * din + j] * h[j];
            z[i] = pic_oracle_act(acc + bk[i], act);
        }
        for (int i = 0; i < dout; ++i) h[i] = z[i];
        p = bk + dout;
    }
    for (int i = 0; i < dims[n_layers - 1]; ++i) f[i] = h[i];
}

/* mu and sigma of the MLP^s output of one image over all its pixels (the
 * encoder's statistics); `work` holds pic_oracle_latent_count doubles.
 * Needs n_layers >= 2.  Returns 0 or -1. */
int pic_oracle_mlps_stats(const int32_t *latents, const double *steps, const double *weights,
                          int L, int C, int n_layers, const int *dims, int act, int H, int W,
                          double *mu, double *sigma, double *work)
{
    double *y[PIC_ORACLE_MAX_LEVELS];
    if (check_args(H, W, L, C, n_layers, dims) != 0 || n_layers < 2) return -1;
    dequant_pyramid(latents, steps, L, C, H, W, work, y);
    int Cf = dims[n_layers - 1];
    double feat[PIC_ORACLE_MAX_WIDTH], f[PIC_ORACLE_MAX_WIDTH];
    double s[PIC_ORACLE_MAX_WIDTH], v[PIC_ORACLE_MAX_WIDTH];
    int64_t N = (int64_t)H * W;
    for (int c = 0; c < Cf; ++c) s[c] = v[c] = 0.0;
    for (int yy = 0; yy < H; ++yy)
        for (int x = 0; x < W; ++x) {
            features_at(y, L, C, H, W, x, yy, feat);
            mlps_at(feat, weights, n_layers, dims, act, f);
            for (int c = 0; c < Cf; ++c) s[c] += f[c];
        }
    for (int c = 0; c < Cf; ++c) mu[c] = s[c] / (double)N;
    for (int yy = 0; yy < H; ++yy)
        for (int x = 0; x < W; ++x) {
            features_at(y, L, C, H, W, x, yy, feat);
            mlps_at(feat, weights, n_layers, dims, act, f);
            for (int c = 0; c < Cf; ++c) v[c] += (f[c] - mu[c]) * (f[c] - mu[c]);
        }
    for (int c = 0; c < Cf; ++c) sigma[c] = sqrt(v[c] / (double)N);
    return 0;
}

/* The un-fused decode: per pixel MLP^s, then normalise and modulate with the
 * given mu, sigma, gamma, beta, then MLP^i (the last layer of `weights`),
 * then clamp.  Returns 0 or -1. */
int pic_oracle_decode_modulated(const int32_t *latents, const double *steps, const double *weights,
                                int L, int C, int n_layers, const int *dims, int act, int clamp,
                                const double *gamma, const double *beta, const double *mu,
                                const double *sigma, int H, int W, double *out_rgb, double *work,
                                int nthreads)
{
    double *y[PIC_ORACLE_MAX_LEVELS];
    if (check_args(H, W, L, C, n_layers, dims) != 0 || n_layers < 2) return -1;
    dequant_pyramid(latents, steps, L, C, H, W, work, y);
    int Cf = dims[n_layers - 1];
    const double *wl = weights;  /* the last layer's W and b */
    for (int k = 0; k < n_layers - 1; ++k) wl += (int64_t)dims[k + 1] * (dims[k] + 1);
    const double *bl = wl + (int64_t)3 * Cf;
    int64_t plane = (int64_t)H * W;
#ifdef _OPENMP
#pragma omp parallel for num_threads(nthreads > 0 ? nthreads : 1) schedule(static)
#endif
    for (int yy = 0; yy < H; ++yy) {
        double feat[PIC_ORACLE_MAX_WIDTH], f[PIC_ORACLE_MAX_WIDTH];
        for (int x = 0; x < W; ++x) {
            features_at(y, L, C, H, W, x, yy, feat);
            mlps_at(feat, weights, n_layers, dims, act, f);
            for (int c = 0; c < Cf; ++c) f[c] = gamma[c] * ((f[c] - mu[c]) / sigma[c]) + beta[c];
            for (int i = 0; i < 3; ++i) {
                double s = 0.0;
                for (int c = 0; c < Cf; ++c) s += wl[(int64_t)i * Cf + c] * f[c];
                s += bl[i];
                out_rgb[i * plane + (int64_t)yy * W + x] = clamp ? pic_oracle_clamp01(s) : s;
            }
        }
    }
    (void)nthreads;
    return 0;
}

/* ------------------------------------------------------------------------
 * Huffman coding of the ZpR symbol stream (Sec. 3.3: image-specific Huffman
 * tables; O(1) decoding per symbol from a table of 2^p entries, p the code
 * precision, i.e. the longest code; the table stored run-length compressed,
 * one entry per coded symbol).
 *
 * Readings:
 *  - the code is a canonical prefix code with lengths <= p, the optimal one
 *    under that limit (package-merge, Larmore & Hirschberg 1990);
 *  - canonical order: symbols sorted by (code length, symbol value); codes
 *    are assigned in that order, each the previous plus one, shifted left
 *    when the length grows.  The stored table is that list of (value,
 *    length); in the 2^p-entry lookup table the k-th symbol covers
 *    2^(p - length) consecutive entries (its run), so the list is the
 *    table's run-length code;
 *  - bits are written most significant first into 32-bit words.
 * The decoder here reads bit by bit against the canonical code (the
 * textbook method), not through the lookup table.
 * ------------------------------------------------------------------------ */

#define PIC_HUFF_MAX_SYMS 4096
#define PIC_HUFF_MAX_LEN 24

/* Optimal code lengths under max_len for n symbols with weights freq (0
 * weight: not coded, length 0).  Package-merge: at each of max_len levels
 * the list is the leaves merged with the pairs (packages) of the previous
 * level's list; a leaf's code length is the number of times it occurs in the
 * first 2m - 2 items of the last list (m coded symbols).  Returns 0, or -1
 * if 2^max_len < m or the arguments are out of range. */
int pic_oracle_huffman_lengths(const int64_t *freq, int n, int max_len, int *len)
{
    if (n < 1 || n > PIC_HUFF_MAX_SYMS || max_len < 1 || max_len > PIC_HUFF_MAX_LEN) return -1;
    int idx[PIC_HUFF_MAX_SYMS], m = 0;
    for (int i = 0; i < n; ++i) {
        len[i] = 0;
        if (freq[i] > 0) idx[m++] = i;
    }
    if (m == 0) return 0;
    if (m == 1) {
        len[idx[0]] = 1;
        return 0;
    }
    if (max_len < 31 && (1LL << max_len) < m) return -1;
    /* leaves sorted by weight (insertion sort; ties by symbol index) */
    for (int a = 1; a < m; ++a) {
        int v = idx[a], b = a - 1;
        while (b >= 0 && (freq[idx[b]] > freq[v] || (freq[idx[b]] == freq[v] && idx[b] > v))) {
            idx[b + 1] = idx[b];
            --b;
        }
        idx[b + 1] = v;
    }
    /* items: weight and either a leaf (child_a < 0, leaf = -child_a - 1) or
     * a package of two items of the previous level */
    static int64_t wt[PIC_HUFF_MAX_LEN + 1][2 * PIC_HUFF_MAX_SYMS];
    static int ca[PIC_HUFF_MAX_LEN + 1][2 * PIC_HUFF_MAX_SYMS];
    static int cnt_lvl[PIC_HUFF_MAX_LEN + 1];
    /* level 1: the leaves */
    for (int a = 0; a < m; ++a) {
        wt[1][a] = freq[idx[a]];
        ca[1][a] = -idx[a] - 1;
    }
    cnt_lvl[1] = m;
    for (int lv = 2; lv <= max_len; ++lv) {
        int np = cnt_lvl[lv - 1] / 2, a = 0, p = 0, k = 0;
        while (a < m || p < np) {
            int64_t wp = p < np ? wt[lv - 1][2 * p] + wt[lv - 1][2 * p + 1] : 0;
            if (p >= np || (a < m && freq[idx[a]] <= wp)) {
                wt[lv][k] = freq[idx[a]];
                ca[lv][k] = -idx[a] - 1;
                ++a;
            } else {
                wt[lv][k] = wp;
                ca[lv][k] = 2 * p; /* children 2p, 2p+1 of level lv - 1 */
                ++p;
            }
            ++k;
        }
        cnt_lvl[lv] = k;
    }
    /* count leaf occurrences in the first 2m - 2 items of the last level */
    static int take[PIC_HUFF_MAX_LEN + 1];
    take[max_len] = 2 * m - 2;
    for (int lv = max_len; lv >= 1; --lv) {
        int packs = 0;
        for (int k = 0; k < take[lv]; ++k) {
            if (ca[lv][k] < 0) len[-ca[lv][k] - 1] += 1;
            else packs += 1;
        }
        if (lv > 1) take[lv - 1] = 2 * packs;
    }
    return 0;
}

/* Canonical order of the coded symbols: order[] receives the indices i with
 * len[i] > 0 sorted by (len, value[i]); returns their number. */
static int canonical_order(const int32_t *value, const int *len, int n, int *order)
{
    int m = 0;
    for (int i = 0; i < n; ++i)
        if (len[i] > 0) order[m++] = i;
    for (int a = 1; a < m; ++a) {
        int v = order[a], b = a - 1;
        while (b >= 0 && (len[order[b]] > len[v] ||
                          (len[order[b]] == len[v] && value[order[b]] > value[v]))) {
            order[b + 1] = order[b];
            --b;
        }
        order[b + 1] = v;
    }
    return m;
}

/* The stored (run-length) table: the coded symbols' values and lengths in
 * canonical order.  Returns the number of entries. */
int pic_oracle_huffman_table(const int32_t *value, const int *len, int n, int32_t *tab_value,
                             int *tab_len)
{
    int order[PIC_HUFF_MAX_SYMS];
    if (n < 1 || n > PIC_HUFF_MAX_SYMS) return -1;
    int m = canonical_order(value, len, n, order);
    for (int k = 0; k < m; ++k) {
        tab_value[k] = value[order[k]];
        tab_len[k] = len[order[k]];
    }
    return m;
}

/* Codes of the table entries in canonical order: code_k = (code_{k-1} + 1)
 * << (len_k - len_{k-1}), code_0 = 0. */
static void canonical_codes(const int *tab_len, int m, uint32_t *code)
{
    uint32_t c = 0;
    for (int k = 0; k < m; ++k) {
        if (k > 0) c = (c + 1) << (tab_len[k] - tab_len[k - 1]);
        code[k] = c;
    }
}

/* Encodes n symbols (values that must be in the table) MSB-first into
 * 32-bit words; returns the number of bits, or -1 (a value not in the
 * table, or cap_words too small). */
int64_t pic_oracle_huffman_encode(const int32_t *syms, int64_t n, const int32_t *tab_value,
                                  const int *tab_len, int m, uint32_t *words, int64_t cap_words)
{
    uint32_t code[PIC_HUFF_MAX_SYMS];
    if (m < 1 || m > PIC_HUFF_MAX_SYMS) return -1;
    canonical_codes(tab_len, m, code);
    for (int64_t w = 0; w < cap_words; ++w) words[w] = 0;
    int64_t bit = 0;
    for (int64_t i = 0; i < n; ++i) {
        int k = 0;
        while (k < m && tab_value[k] != syms[i]) ++k;
        if (k == m) return -1;
        for (int b = tab_len[k] - 1; b >= 0; --b) {
            if ((bit >> 5) >= cap_words) return -1;
            if ((code[k] >> b) & 1u) words[bit >> 5] |= 0x80000000u >> (bit & 31);
            ++bit;
        }
    }
    return bit;
}

/* Decodes n_out symbols from n_bits bits: reads one bit at a time, and
 * after every bit checks whether the code read so far is a codeword of the
 * current length (canonical decoding).  Returns 0, or -1 if the bits run out
 * or end inside a codeword that is not complete. */
int pic_oracle_huffman_decode(const uint32_t *words, int64_t n_bits, const int32_t *tab_value,
                              const int *tab_len, int m, int32_t *out, int64_t n_out)
{
    uint32_t code[PIC_HUFF_MAX_SYMS];
    if (m < 1 || m > PIC_HUFF_MAX_SYMS) return -1;
    canonical_codes(tab_len, m, code);
    int64_t bit = 0;
    for (int64_t i = 0; i < n_out; ++i) {
        uint32_t c = 0;
        int l = 0, found = -1;
        while (found < 0) {
            if (bit >= n_bits || l >= PIC_HUFF_MAX_LEN) return -1;
            c = (c << 1) | ((words[bit >> 5] >> (31 - (bit & 31))) & 1u);
            ++bit;
            ++l;
            for (int k = 0; k < m; ++k)
                if (tab_len[k] == l && code[k] == c) {
                    found = k;
                    break;
                }
        }
        out[i] = tab_value[found];
    }
    return bit == n_bits ? 0 : -1;
}
