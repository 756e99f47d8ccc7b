// k_idct.cu -- inverse DCT stage (include/pic_idct.h): dequantise the 8x8
// DCT coefficient patches of every latent plane, inverse-transform them and
// put them back into the latent pyramid (Fig. 1; Sec. 3.2, Eqs. 5-7 run
// backwards).
//
// The stage is bound by HBM: per patch it reads 256 B of int32 coefficients
// and writes up to 256 B of fp32 latents, against 2 x 512 FMAs of the
// separable transform (done as butterflies, below).  One CTA pass takes 32
// consecutive patches, 8 threads
// per patch (the 8 threads of a patch sit in one warp, so the exchanges
// between the two 1-D passes need only __syncwarp):
//   load    thread j reads 16 B at coefficient 4j and 32 + 4j of its patch
//           (a warp reads 4 whole patches, 1 KB contiguous) one pass ahead,
//           scales them by the level's step and stores them into the
//           patch's shared slot;
//   pass 1  thread j transforms column j: T[m][j] = sum_u c[u][m] S[u][j];
//   pass 2  thread j transforms row j:    x[j][n] = sum_v c[v][n] T[j][v];
//   store   lanes 2i and 2i+1 trade row halves so that each store
//           instruction writes whole 32-byte rows: row 2i in the first,
//           row 2i+1 in the second.
// Each 1-D transform x[n] = sum_k a(k) X[k] cos((2n + 1) k pi / 16) is the
// even/odd split of the basis (cos((2(7-n) + 1) k pi / 16) = (-1)^k times
// that of n): x[n] = E[n] + O[n], x[7-n] = E[n] - O[n] with E the 4-point
// transform of X[0, 2, 4, 6] (split once more) and O a 4x4 product of
// X[1, 3, 5, 7] -- 36 operations instead of 64 multiply-adds.  The patch
// slot is padded to 72 floats so the column accesses of pass 1 hit 32
// distinct banks.
#include <cstdint>

#include <cuda_runtime.h>

#include "pic_decode.h"
#include "pic_idct.h"

namespace {

constexpr int kLevelsMax = 12;
constexpr int kChanMax = 4;
constexpr int kPlanesMax = kLevelsMax * kChanMax;
constexpr int kThreads = 256;
constexpr int kPatches = kThreads / 8;  // patches per CTA pass
constexpr int kSlot = 72;               // floats per patch slot (64 + 8 bank pad)

struct Plane {
  int blk0;                     // first patch of the plane, counted within one image
  int bw;                       // patches per row: ceil(W_l / 8)
  unsigned long long bw_inv;    // division by bw (see udiv)
  long long lat_off;            // offset of the plane within one image's latents
  int Hl, Wl;
  int level;
};

struct IdctParams {
  const int32_t* coeffs;
  const float* steps;
  float* latents;
  int blocks_per_image;
  unsigned long long bpi_inv;   // division by blocks_per_image
  long long lat_per_image;
  int total_blocks;             // < 2^31
  int L, n_planes;
  Plane pl[kPlanesMax];
};

// 0.5 cos(k pi / 16), k = 1 .. 7 (k = 4 is also a(0) = 1 / sqrt(8))
constexpr float kC1 = 4.903926402e-01f, kC2 = 4.619397663e-01f, kC3 = 4.157348062e-01f,
                kC4 = 3.535533906e-01f, kC5 = 2.777851165e-01f, kC6 = 1.913417162e-01f,
                kC7 = 9.754516101e-02f;

// 8-point inverse DCT of X (frequencies) into x (samples), by the split above.
__device__ __forceinline__ void idct8(const float (&X)[8], float (&x)[8]) {
  const float ee0 = kC4 * (X[0] + X[4]), ee1 = kC4 * (X[0] - X[4]);
  const float eo0 = fmaf(kC2, X[2], kC6 * X[6]), eo1 = fmaf(kC6, X[2], -kC2 * X[6]);
  const float e0 = ee0 + eo0, e3 = ee0 - eo0, e1 = ee1 + eo1, e2 = ee1 - eo1;
  const float o0 = fmaf(kC1, X[1], fmaf(kC3, X[3], fmaf(kC5, X[5], kC7 * X[7])));
  const float o1 = fmaf(kC3, X[1], fmaf(-kC7, X[3], fmaf(-kC1, X[5], -kC5 * X[7])));
  const float o2 = fmaf(kC5, X[1], fmaf(-kC1, X[3], fmaf(kC7, X[5], kC3 * X[7])));
  const float o3 = fmaf(kC7, X[1], fmaf(-kC5, X[3], fmaf(kC3, X[5], -kC1 * X[7])));
  x[0] = e0 + o0;
  x[7] = e0 - o0;
  x[1] = e1 + o1;
  x[6] = e1 - o1;
  x[2] = e2 + o2;
  x[5] = e2 - o2;
  x[3] = e3 + o3;
  x[4] = e3 - o3;
}

// floor(n / d) for 32-bit n and d by one multiply-high with inv = ceil(2^64 / d)
// (division by invariant integers, Granlund & Montgomery 1994: the error term
// n (inv d - 2^64) / (d 2^64) stays below 1/d); d == 1 is stored as inv == 0.
__host__ unsigned long long udiv_inv(unsigned d) { return d > 1 ? ~0ULL / d + 1 : 0; }
__device__ __forceinline__ unsigned udiv(unsigned n, unsigned d, unsigned long long inv) {
  (void)d;
  return inv ? static_cast<unsigned>(__umul64hi(n, inv)) : n;
}

int level_size(int n, int l) { return static_cast<int>((static_cast<long long>(n) + (1LL << l) - 1) >> l); }

__global__ void __launch_bounds__(kThreads, 6)
    idct_unpatchify_kernel(const __grid_constant__ IdctParams p) {
  __shared__ __align__(16) float tile[kPatches * kSlot];
  const int t = threadIdx.x;
  const int slot = t >> 3;
  const int j = t & 7;
  const int odd = j & 1;
  float* my = tile + slot * kSlot;

  const int stride = static_cast<int>(gridDim.x) * kPatches;
  int g = static_cast<int>(blockIdx.x) * kPatches + slot;
  int4 v0 = make_int4(0, 0, 0, 0), v1 = v0;
  if (g < p.total_blocks) {
    const int4* src = reinterpret_cast<const int4*>(p.coeffs + static_cast<long long>(g) * 64);
    v0 = __ldcs(src + j);
    v1 = __ldcs(src + 8 + j);
  }
  for (int g0 = static_cast<int>(blockIdx.x) * kPatches; g0 < p.total_blocks;
       g0 += stride, g += stride) {
    const bool live = g < p.total_blocks;
    int4 n0 = make_int4(0, 0, 0, 0), n1 = n0;
    if (g + stride < p.total_blocks) {  // next pass's coefficients
      const int4* src = reinterpret_cast<const int4*>(p.coeffs + static_cast<long long>(g + stride) * 64);
      n0 = __ldcs(src + j);
      n1 = __ldcs(src + 8 + j);
    }
    int b = 0, k = 0, pi = 0;
    float step = 0.0f;
    if (live) {
      b = static_cast<int>(udiv(g, p.blocks_per_image, p.bpi_inv));
      k = g - b * p.blocks_per_image;
      int hi = p.n_planes - 1;  // last plane whose first patch is <= k
      while (pi < hi) {
        const int mid = (pi + hi + 1) >> 1;
        if (k >= p.pl[mid].blk0) pi = mid;
        else hi = mid - 1;
      }
      step = __ldg(p.steps + b * p.L + p.pl[pi].level);
    }
    reinterpret_cast<float4*>(my)[j] =
        make_float4(v0.x * step, v0.y * step, v0.z * step, v0.w * step);
    reinterpret_cast<float4*>(my + 32)[j] =
        make_float4(v1.x * step, v1.y * step, v1.z * step, v1.w * step);
    v0 = n0;
    v1 = n1;
    __syncwarp();

    // pass 1: column j, vertical inverse transform
    float col[8], tr[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) col[u] = my[u * 8 + j];
    idct8(col, tr);
    __syncwarp();
#pragma unroll
    for (int m = 0; m < 8; ++m) my[m * 8 + j] = tr[m];
    __syncwarp();

    // pass 2: row j, horizontal inverse transform
    const float4 r0 = reinterpret_cast<const float4*>(my)[2 * j];
    const float4 r1 = reinterpret_cast<const float4*>(my)[2 * j + 1];
    const float row[8] = {r0.x, r0.y, r0.z, r0.w, r1.x, r1.y, r1.z, r1.w};
    float x[8];
    idct8(row, x);
    __syncwarp();  // the slot is refilled by the next pass

    // lanes 2i, 2i+1: the even lane sends its right half, the odd lane its left
    float recv[4];
#pragma unroll
    for (int n = 0; n < 4; ++n) recv[n] = __shfl_xor_sync(0xffffffffu, odd ? x[n] : x[4 + n], 1);
    // store 0 writes row j & ~1 (even lane: columns 0-3 of its own row; odd
    // lane: columns 4-7 received), store 1 row j | 1 (even lane: columns 0-3
    // received; odd lane: columns 4-7 of its own row)
    const float4 s0 = odd ? make_float4(recv[0], recv[1], recv[2], recv[3])
                          : make_float4(x[0], x[1], x[2], x[3]);
    const float4 s1 = odd ? make_float4(x[4], x[5], x[6], x[7])
                          : make_float4(recv[0], recv[1], recv[2], recv[3]);
    if (live) {
      const Plane& P = p.pl[pi];
      const int pr = k - P.blk0;
      const int by = static_cast<int>(udiv(pr, P.bw, P.bw_inv)), bx = pr - by * P.bw;
      const int q0 = 8 * bx + 4 * odd;
      const int nv = min(4, P.Wl - q0);  // valid columns of this half (may be <= 0)
      float* plane = p.latents + b * p.lat_per_image + P.lat_off + q0;
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int r = 8 * by + (e ? (j | 1) : (j & ~1));
        const float4 sv = e ? s1 : s0;
        if (r < P.Hl && nv > 0) {
          float* dst = plane + static_cast<long long>(r) * P.Wl;
          if (nv == 4 && (reinterpret_cast<uintptr_t>(dst) & 15u) == 0) {
            *reinterpret_cast<float4*>(dst) = sv;
          } else {
            const float vv[4] = {sv.x, sv.y, sv.z, sv.w};
#pragma unroll
            for (int n = 0; n < 4; ++n)
              if (n < nv) dst[n] = vv[n];
          }
        }
      }
    }
  }
}

bool sizes_ok(int H, int W, int L, int C) {
  return H >= 1 && W >= 1 && H <= 65536 && W <= 65536 && L >= 1 && L <= kLevelsMax && C >= 1 &&
         C <= kChanMax;
}

}  // namespace

extern "C" int64_t pic_idct_block_count(int H, int W, int L, int C) {
  if (!sizes_ok(H, W, L, C)) return -1;
  int64_t n = 0;
  for (int l = 0; l < L; ++l)
    n += static_cast<int64_t>(C) * ((level_size(H, l) + 7) / 8) * ((level_size(W, l) + 7) / 8);
  return n;
}

extern "C" int pic_idct_unpatchify(const int32_t* coeffs, const float* steps, int B, int H, int W,
                                   int L, int C, float* latents, void* stream) {
  if (!coeffs || !steps || !latents || B < 1 || B > 65536 || !sizes_ok(H, W, L, C))
    return PIC_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(coeffs) & 15u) != 0 ||
      (reinterpret_cast<uintptr_t>(latents) & 3u) != 0 ||
      (reinterpret_cast<uintptr_t>(steps) & 3u) != 0)
    return PIC_ERR_INVALID_ARG;
  IdctParams p{};
  p.coeffs = coeffs;
  p.steps = steps;
  p.latents = latents;
  p.L = L;
  long long blk = 0, off = 0;
  int q = 0;
  for (int l = 0; l < L; ++l) {
    const int Hl = level_size(H, l), Wl = level_size(W, l);
    for (int c = 0; c < C; ++c, ++q) {
      Plane& P = p.pl[q];
      P.blk0 = static_cast<int>(blk);
      P.lat_off = off + static_cast<long long>(c) * Hl * Wl;
      P.bw = (Wl + 7) / 8;
      P.bw_inv = udiv_inv(static_cast<unsigned>(P.bw));
      P.Hl = Hl;
      P.Wl = Wl;
      P.level = l;
      blk += static_cast<long long>(P.bw) * ((Hl + 7) / 8);
    }
    off += static_cast<long long>(C) * Hl * Wl;
  }
  if (blk * B >= (1LL << 31) - (1LL << 24)) return PIC_ERR_INVALID_ARG;  // 32-bit patch indices (+ one stride)
  p.n_planes = q;
  p.blocks_per_image = static_cast<int>(blk);
  p.bpi_inv = udiv_inv(static_cast<unsigned>(blk));
  p.lat_per_image = off;
  p.total_blocks = static_cast<int>(blk * B);

  int dev = 0, sms = 0, per_sm = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, idct_unpatchify_kernel, kThreads, 0) !=
          cudaSuccess) {
    cudaGetLastError();
    return PIC_ERR_CUDA;
  }
  const long long passes = (p.total_blocks + kPatches - 1) / kPatches;
  const long long cap = static_cast<long long>(sms) * (per_sm > 0 ? per_sm : 1);
  const unsigned grid = static_cast<unsigned>(passes < cap ? passes : cap);
  idct_unpatchify_kernel<<<grid, kThreads, 0, static_cast<cudaStream_t>(stream)>>>(p);
  if (cudaGetLastError() != cudaSuccess) return PIC_ERR_CUDA;
  return PIC_OK;
}
