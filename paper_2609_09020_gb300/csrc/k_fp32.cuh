// k_fp32.cuh -- the fp32 CUDA-core decode kernel templates (PIC_PREC_FP32),
// instantiated in k_fp32.cu (the decode workloads' architectures, the
// generic kernel, the registry) and k_fp32_sweep.cu (the width ablation).
//
// The decode fused on the fp32 CUDA cores.
//
// One thread decodes one pixel: dequantisation and bilinear upsampling of
// every pyramid level (Sec. 3.1, Eq. 1) straight into registers, the
// synthesis MLP g_s (Sec. 4.1) with the layer dims fixed at compile time, and
// the clamped planar RGB store.  Features and hidden activations never leave
// the registers.  The MLP runs on packed f32x2 FMAs: one instruction does two
// output neurons, so the FMA pipe stays full while half the issue slots
// remain for the shared-memory weight loads (broadcast LDS.128) and the rest.
//
// Work split: a tile is 128 consecutive pixels of one image row; the tiles of
// all images are numbered image-major and each CTA takes one contiguous range
// of them (so a CTA sees at most a couple of images and loads each image's
// weights into shared memory once).  Grid = resident CTAs over all SMs.

#pragma once

#include "pic_common.cuh"
#include "pic_kernels.h"

namespace pic {
namespace {

constexpr int kThreads = 128;

__host__ __device__ constexpr int round4(int d) { return (d + 3) & ~3; }

// Shared-memory image of one layer: W^T [din][round4(dout)] then the bias
// [round4(dout)], zero padded.  Floats per layer:
__host__ __device__ constexpr int layer_floats(int din, int dout) {
  return (din + 1) * round4(dout);
}

// Copies one layer's weights from the nn.Linear layout (W [dout][din]
// row-major, then b) into its transposed, padded shared-memory image.
__device__ __forceinline__ void load_layer_fp32(float* __restrict__ sm, const float* __restrict__ w,
                                                int din, int dout) {
  const int d4 = round4(dout);
  const int n = (din + 1) * d4;
  for (int e = threadIdx.x; e < n; e += blockDim.x) {
    const int j = e / d4, i = e - j * d4;  // row j of W^T (j == din: the bias row), column i
    float v = 0.0f;
    if (i < dout) v = (j < din) ? w[i * din + j] : w[dout * din + i];
    sm[e] = v;
  }
}

template <int NL, int D0, int D1, int D2, int D3, int D4>
__device__ __forceinline__ void load_weights_fp32(float* __restrict__ sm, const float* __restrict__ w) {
  load_layer_fp32(sm, w, D0, D1);
  sm += layer_floats(D0, D1);
  w += D1 * D0 + D1;
  if constexpr (NL >= 2) {
    load_layer_fp32(sm, w, D1, D2);
    sm += layer_floats(D1, D2);
    w += D2 * D1 + D2;
  }
  if constexpr (NL >= 3) {
    load_layer_fp32(sm, w, D2, D3);
    sm += layer_floats(D2, D3);
    w += D3 * D2 + D3;
  }
  if constexpr (NL >= 4) load_layer_fp32(sm, w, D3, D4);
}

// out = act(W in + b) (or W in + b for the last layer), packed-pair FMAs.
// `wt` is the layer's shared-memory image.
template <int DIN, int DOUT, int ACT, bool LAST, int MAXW>
__device__ __forceinline__ void dense_layer(const float* __restrict__ wt, const float (&in)[MAXW],
                                            float (&out)[MAXW]) {
  constexpr int D4 = round4(DOUT);
  unsigned long long acc[D4 / 2];
  const float* bias = wt + DIN * D4;
#pragma unroll
  for (int i = 0; i < D4 / 4; ++i) {
    const ulonglong2 b = *reinterpret_cast<const ulonglong2*>(bias + 4 * i);
    acc[2 * i] = b.x;
    acc[2 * i + 1] = b.y;
  }
#pragma unroll
  for (int j = 0; j < DIN; ++j) {
    const unsigned long long hh = pack2(in[j], in[j]);
#pragma unroll
    for (int i = 0; i < D4 / 4; ++i) {
      const ulonglong2 w = *reinterpret_cast<const ulonglong2*>(wt + j * D4 + 4 * i);
      acc[2 * i] = fma2(w.x, hh, acc[2 * i]);
      acc[2 * i + 1] = fma2(w.y, hh, acc[2 * i + 1]);
    }
  }
#pragma unroll
  for (int i = 0; i < D4 / 2; ++i) {
    if constexpr (ACT == ACT_GELU && !LAST) acc[i] = gelu_poly2(acc[i]);
    const float2 v = unpack2(acc[i]);
    if constexpr (LAST || ACT == ACT_GELU) {
      if (2 * i < DOUT) out[2 * i] = v.x;
      if (2 * i + 1 < DOUT) out[2 * i + 1] = v.y;
    } else {
      if (2 * i < DOUT) out[2 * i] = activate<ACT>(v.x);
      if (2 * i + 1 < DOUT) out[2 * i + 1] = activate<ACT>(v.y);
    }
  }
}

template <int C, int NL, int D0, int D1, int D2, int D3, int D4, int ACT>
struct Fp32Net {
  static constexpr int L = D0 / C;
  static constexpr int MAXW = (D0 > D1 ? D0 : D1) > (D2 > D3 ? D2 : D3)
                                  ? (D0 > D1 ? D0 : D1)
                                  : (D2 > D3 ? D2 : D3);
  static constexpr int W_ = MAXW > D4 ? MAXW : D4;
  static constexpr int smem_floats() {
    int n = layer_floats(D0, D1);
    if (NL >= 2) n += layer_floats(D1, D2);
    if (NL >= 3) n += layer_floats(D2, D3);
    if (NL >= 4) n += layer_floats(D3, D4);
    return n;
  }
};

template <int C, int NL, int D0, int D1, int D2, int D3, int D4, int ACT, bool FL>
__global__ void __launch_bounds__(kThreads)
    fp32_decode_kernel(const DecodeParams p) {
  using Net = Fp32Net<C, NL, D0, D1, D2, D3, D4, ACT>;
  constexpr int L = Net::L;
  constexpr int MW = Net::W_;
  extern __shared__ __align__(16) float sm_w[];

  const long long chunk = (p.total_tiles + gridDim.x - 1) / gridDim.x;
  const long long t_begin = blockIdx.x * chunk;
  const long long t_end = min(t_begin + chunk, p.total_tiles);
  const float* wts = static_cast<const float*>(p.weights);
  const long long plane = static_cast<long long>(p.H) * p.W;
  int cur_b = -1;
  float step[L];

  for (long long t = t_begin; t < t_end; ++t) {
    const int b = static_cast<int>(t / p.tiles_per_image);
    const long long r = t - static_cast<long long>(b) * p.tiles_per_image;
    const int y = static_cast<int>(r / p.tiles_per_row);
    const int x = static_cast<int>(r - static_cast<long long>(y) * p.tiles_per_row) * kThreads +
                  threadIdx.x;
    if (b != cur_b) {  // uniform across the CTA
      __syncthreads();
      load_weights_fp32<NL, D0, D1, D2, D3, D4>(sm_w, wts + b * p.params_per_image);
      __syncthreads();
#pragma unroll
      for (int l = 0; l < L; ++l) step[l] = FL ? 1.0f : __ldg(p.steps + b * L + l);
      cur_b = b;
    }
    if (x >= p.W) continue;

    // ---- steps 1-3: dequantise, upsample and concatenate every level ----
    const int32_t* lat = p.latents + b * p.lat_per_image;
    float h[MW], g[MW];
#pragma unroll
    for (int l = 0; l < L; ++l) {
      const LevelGeom lg = p.lv[l];
      if (l == 0) {  // level 0 has the output size: the upsampling is the identity
#pragma unroll
        for (int c = 0; c < C; ++c)
          h[c] = step[0] * lat_value<FL>(__ldg(lat + c * plane + static_cast<long long>(y) * p.W + x));
      } else {
        const Tap tx = bilinear_tap(x, lg.sx, lg.W);
        const Tap ty = bilinear_tap(y, lg.sy, lg.H);
#pragma unroll
        for (int c = 0; c < C; ++c)
          h[l * C + c] = step[l] * bilinear_sample<FL>(lat + lg.off + static_cast<long long>(c) * lg.H * lg.W,
                                                   lg.W, tx, ty);
      }
    }

    // ---- step 4: the synthesis MLP (ping-pong between h and g) ----
    const float* wl = sm_w;
    float rgb[3];
    dense_layer<D0, D1, ACT, NL == 1>(wl, h, g);
    wl += layer_floats(D0, D1);
    if constexpr (NL == 1) {
      rgb[0] = g[0]; rgb[1] = g[1]; rgb[2] = g[2];
    }
    if constexpr (NL >= 2) {
      dense_layer<D1, D2, ACT, NL == 2>(wl, g, h);
      wl += layer_floats(D1, D2);
      if constexpr (NL == 2) {
        rgb[0] = h[0]; rgb[1] = h[1]; rgb[2] = h[2];
      }
    }
    if constexpr (NL >= 3) {
      dense_layer<D2, D3, ACT, NL == 3>(wl, h, g);
      wl += layer_floats(D2, D3);
      if constexpr (NL == 3) {
        rgb[0] = g[0]; rgb[1] = g[1]; rgb[2] = g[2];
      }
    }
    if constexpr (NL >= 4) {
      dense_layer<D3, D4, ACT, NL == 4>(wl, g, h);
      rgb[0] = h[0]; rgb[1] = h[1]; rgb[2] = h[2];
    }

    // ---- step 5: clamp and store (planar rows are coalesced) ----
    store_rgb(p, b, y, x, rgb[0], rgb[1], rgb[2]);
  }
}

// ---------------------------------------------------------------------------
// Generic kernel: any dims up to kMaxDim, runtime loops, weights in shared
// memory in the nn.Linear layout.  Slower (hidden values in local memory) but
// covers every arch the C ABI accepts.
template <bool FL>
__global__ void __launch_bounds__(kThreads) fp32_generic_kernel(const DecodeParams p) {
  extern __shared__ __align__(16) float sm_w[];
  const long long chunk = (p.total_tiles + gridDim.x - 1) / gridDim.x;
  const long long t_begin = blockIdx.x * chunk;
  const long long t_end = min(t_begin + chunk, p.total_tiles);
  const float* wts = static_cast<const float*>(p.weights);
  int cur_b = -1;
  for (long long t = t_begin; t < t_end; ++t) {
    const int b = static_cast<int>(t / p.tiles_per_image);
    const long long r = t - static_cast<long long>(b) * p.tiles_per_image;
    const int y = static_cast<int>(r / p.tiles_per_row);
    const int x = static_cast<int>(r - static_cast<long long>(y) * p.tiles_per_row) * kThreads +
                  threadIdx.x;
    if (b != cur_b) {
      __syncthreads();
      for (long long e = threadIdx.x; e < p.params_per_image; e += blockDim.x)
        sm_w[e] = wts[b * p.params_per_image + e];
      __syncthreads();
      cur_b = b;
    }
    if (x >= p.W) continue;
    const int32_t* lat = p.latents + b * p.lat_per_image;
    float h[kMaxDim], g[kMaxDim];
    for (int l = 0; l < p.L; ++l) {
      const LevelGeom lg = p.lv[l];
      const float s = FL ? 1.0f : __ldg(p.steps + b * p.L + l);
      const Tap tx = bilinear_tap(x, lg.sx, lg.W);
      const Tap ty = bilinear_tap(y, lg.sy, lg.H);
      for (int c = 0; c < p.C; ++c)
        h[l * p.C + c] = s * bilinear_sample<FL>(lat + lg.off + static_cast<long long>(c) * lg.H * lg.W,
                                             lg.W, tx, ty);
    }
    const float* wl = sm_w;
    for (int k = 0; k < p.n_layers; ++k) {
      const int din = p.dims[k], dout = p.dims[k + 1];
      const bool last = (k == p.n_layers - 1);
      for (int i = 0; i < dout; ++i) {
        float s = wl[dout * din + i];
        for (int j = 0; j < din; ++j) s = fmaf(wl[i * din + j], h[j], s);
        g[i] = last ? s : activate_rt(s, p.act);
      }
      for (int i = 0; i < dout; ++i) h[i] = g[i];
      wl += dout * din + dout;
    }
    store_rgb(p, b, y, x, h[0], h[1], h[2]);
  }
}

template <int C, int NL, int D0, int D1, int D2, int D3, int D4, int ACT, bool FL = false>
KernelInfo make_fp32(const char* name) {
  using Net = Fp32Net<C, NL, D0, D1, D2, D3, D4, ACT>;
  KernelInfo k{};
  k.name = name;
  k.precision = 0;
  k.latent_format = FL ? 1 : 0;
  k.C = C;
  k.n_layers = NL;
  const int d[5] = {D0, D1, D2, D3, D4};
  for (int i = 0; i <= NL; ++i) k.dims[i] = d[i];
  k.act = ACT;
  k.threads = kThreads;
  k.tile_px = kThreads;
  k.smem_bytes = Net::smem_floats() * 4;
  k.fn = reinterpret_cast<const void*>(&fp32_decode_kernel<C, NL, D0, D1, D2, D3, D4, ACT, FL>);
  return k;
}

}  // namespace
}  // namespace pic
