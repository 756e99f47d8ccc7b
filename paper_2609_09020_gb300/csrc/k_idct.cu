// k_idct.cu -- inverse DCT stage (include/pic_idct.h): dequantise the 8x8
// DCT coefficient patches of every latent plane, inverse-transform them and
// put them back into the latent pyramid (Fig. 1; Sec. 3.2, Eqs. 5-7 run
// backwards).
//
// The stage is bound by HBM: per patch it reads 256 B of int32 coefficients
// and writes up to 256 B of fp32 latents, against 2 x 512 FMAs of the
// separable transform.  One CTA pass takes 32 consecutive patches, 8 threads
// per patch (the 8 threads of a patch sit in one warp, so the exchanges
// between the two 1-D passes need only __syncwarp):
//   load    thread j reads 16 B at coefficient 4j and 32 + 4j of its patch
//           (a warp reads 4 whole patches, 1 KB contiguous), scales them by
//           the level's step and stores them into the patch's shared slot;
//   pass 1  thread j transforms column j: T[m][j] = sum_u c[u][m] S[u][j];
//   pass 2  thread j transforms row j:    x[j][n] = sum_v c[v][n] T[j][v];
//   store   thread j writes row j of the patch (32 B, two float4 when the
//           row is whole and aligned) into its plane.
// c[k][n] = a(k) cos((2n + 1) k pi / 16) is built once per CTA in shared
// memory from CUDA's cospi in double precision.  The patch slot is padded to
// 72 floats so the column accesses of pass 1 hit 32 distinct banks.
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
  long long blk0;     // first patch of the plane, counted within one image
  long long lat_off;  // offset of the plane within one image's latents
  int bw;             // patches per row: ceil(W_l / 8)
  int Hl, Wl;
  int level;
};

struct IdctParams {
  const int32_t* coeffs;
  const float* steps;
  float* latents;
  long long blocks_per_image;
  long long lat_per_image;
  long long total_blocks;
  int L, n_planes;
  Plane pl[kPlanesMax];
};

int level_size(int n, int l) { return static_cast<int>((static_cast<long long>(n) + (1LL << l) - 1) >> l); }

__global__ void __launch_bounds__(kThreads)
    idct_unpatchify_kernel(const __grid_constant__ IdctParams p) {
  __shared__ __align__(16) float basis[64];  // basis[k * 8 + n] = a(k) cos((2n+1) k pi / 16)
  __shared__ __align__(16) float tile[kPatches * kSlot];
  const int t = threadIdx.x;
  if (t < 64) {
    const int k = t >> 3, n = t & 7;
    const double a = k == 0 ? rsqrt(8.0) : 0.5;
    basis[t] = static_cast<float>(a * cospi(static_cast<double>((2 * n + 1) * k) / 16.0));
  }
  __syncthreads();
  const int slot = t >> 3;
  const int j = t & 7;
  float* my = tile + slot * kSlot;
  const float4* basis4 = reinterpret_cast<const float4*>(basis);

  for (long long g0 = static_cast<long long>(blockIdx.x) * kPatches; g0 < p.total_blocks;
       g0 += static_cast<long long>(gridDim.x) * kPatches) {
    const long long g = g0 + slot;
    const bool live = g < p.total_blocks;
    int b = 0, pi = 0;
    long long k = 0;
    float step = 0.0f;
    if (live) {
      b = static_cast<int>(g / p.blocks_per_image);
      k = g - static_cast<long long>(b) * p.blocks_per_image;
      for (int q = 1; q < p.n_planes; ++q)
        if (k >= p.pl[q].blk0) pi = q;
      step = __ldg(p.steps + b * p.L + p.pl[pi].level);
      const int4* src = reinterpret_cast<const int4*>(p.coeffs + g * 64);
      const int4 v0 = __ldcs(src + j), v1 = __ldcs(src + 8 + j);
      reinterpret_cast<float4*>(my)[j] =
          make_float4(v0.x * step, v0.y * step, v0.z * step, v0.w * step);
      reinterpret_cast<float4*>(my + 32)[j] =
          make_float4(v1.x * step, v1.y * step, v1.z * step, v1.w * step);
    }
    __syncwarp();

    // pass 1: column j, vertical inverse transform
    float col[8], tr[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) col[u] = my[u * 8 + j];
#pragma unroll
    for (int m = 0; m < 8; ++m) tr[m] = 0.0f;
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const float4 c0 = basis4[2 * u], c1 = basis4[2 * u + 1];
      tr[0] = fmaf(c0.x, col[u], tr[0]);
      tr[1] = fmaf(c0.y, col[u], tr[1]);
      tr[2] = fmaf(c0.z, col[u], tr[2]);
      tr[3] = fmaf(c0.w, col[u], tr[3]);
      tr[4] = fmaf(c1.x, col[u], tr[4]);
      tr[5] = fmaf(c1.y, col[u], tr[5]);
      tr[6] = fmaf(c1.z, col[u], tr[6]);
      tr[7] = fmaf(c1.w, col[u], tr[7]);
    }
    __syncwarp();
#pragma unroll
    for (int m = 0; m < 8; ++m) my[m * 8 + j] = tr[m];
    __syncwarp();

    // pass 2: row j, horizontal inverse transform
    const float4 r0 = reinterpret_cast<const float4*>(my)[2 * j];
    const float4 r1 = reinterpret_cast<const float4*>(my)[2 * j + 1];
    const float row[8] = {r0.x, r0.y, r0.z, r0.w, r1.x, r1.y, r1.z, r1.w};
    float x[8];
#pragma unroll
    for (int n = 0; n < 8; ++n) x[n] = 0.0f;
#pragma unroll
    for (int v = 0; v < 8; ++v) {
      const float4 c0 = basis4[2 * v], c1 = basis4[2 * v + 1];
      x[0] = fmaf(c0.x, row[v], x[0]);
      x[1] = fmaf(c0.y, row[v], x[1]);
      x[2] = fmaf(c0.z, row[v], x[2]);
      x[3] = fmaf(c0.w, row[v], x[3]);
      x[4] = fmaf(c1.x, row[v], x[4]);
      x[5] = fmaf(c1.y, row[v], x[5]);
      x[6] = fmaf(c1.z, row[v], x[6]);
      x[7] = fmaf(c1.w, row[v], x[7]);
    }
    __syncwarp();  // the slot is refilled by the next pass

    if (live) {
      const Plane& P = p.pl[pi];
      const int pr = static_cast<int>(k - P.blk0);
      const int by = pr / P.bw, bx = pr - by * P.bw;
      const int r = 8 * by + j;
      if (r < P.Hl) {
        const int q0 = 8 * bx;
        float* dst = p.latents + b * p.lat_per_image + P.lat_off + static_cast<long long>(r) * P.Wl + q0;
        const int nv = min(8, P.Wl - q0);
        if (nv == 8 && (reinterpret_cast<uintptr_t>(dst) & 15u) == 0) {
          reinterpret_cast<float4*>(dst)[0] = make_float4(x[0], x[1], x[2], x[3]);
          reinterpret_cast<float4*>(dst)[1] = make_float4(x[4], x[5], x[6], x[7]);
        } else {
#pragma unroll
          for (int n = 0; n < 8; ++n)
            if (n < nv) dst[n] = x[n];
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
      P.blk0 = blk;
      P.lat_off = off + static_cast<long long>(c) * Hl * Wl;
      P.bw = (Wl + 7) / 8;
      P.Hl = Hl;
      P.Wl = Wl;
      P.level = l;
      blk += static_cast<long long>(P.bw) * ((Hl + 7) / 8);
    }
    off += static_cast<long long>(C) * Hl * Wl;
  }
  p.n_planes = q;
  p.blocks_per_image = blk;
  p.lat_per_image = off;
  p.total_blocks = blk * B;

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
