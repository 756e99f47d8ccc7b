// k_fp32.cuh -- the fp32 CUDA-core decode kernel templates (PIC_PREC_FP32),
// instantiated in k_fp32.cu (the decode workloads' architectures, the
// generic kernel, the registry) and k_fp32_sweep.cu (the width ablation).
//
// The decode fused on the fp32 CUDA cores.
//
// A CTA of 128 threads decodes tiles of 128 consecutive pixels of one image
// row.  Per tile:
//   1. features: thread p dequantises and upsamples every pyramid level for
//      pixel p (Sec. 3.1, Eq. 1) and writes the feature vector into a
//      shared-memory activation buffer X (one row of 128 floats per
//      feature), so features never reach HBM;
//   2. each hidden layer of g_s (Sec. 4.1) is a 128-pixel x N contraction
//      on the CUDA cores, register-tiled: thread (pg, ng) accumulates TP
//      pixels x TN neurons (TP = NG, NG x TN = N; 8 x 8 for N = 64) over the
//      K inputs, reading TP activations and TN weights from shared memory
//      per input, so one load feeds TN (resp. TP) FMAs instead of one;
//      packed f32x2 FMAs do two neurons of one pixel per instruction.  The
//      bias seeds the accumulators; the activation is applied in registers
//      and the layer's output rows are written back over X;
//   3. the output layer (3 neurons) is folded into the last hidden layer's
//      epilogue: each thread forms the 3 partial sums over its TN neurons for
//      its TP pixels, and thread p adds the NG partials of pixel p, the bias,
//      clamps and stores the planar RGB row (coalesced).
// Weights live in shared memory for the whole tile range (reloaded when the
// image changes).  Activation rows are 16-byte chunks XOR-swizzled by the
// writing thread's neuron group, so the epilogue stores and the K-loop loads
// both run without bank conflicts.
//
// Work split: the tiles of all images are numbered image-major and each CTA
// takes one contiguous range of them (a CTA sees at most a couple of images
// and loads each one's weights once).  Grid = resident CTAs over all SMs.

#pragma once

#include "pic_common.cuh"
#include "pic_kernels.h"

namespace pic {
namespace {

constexpr int kThreads = 128;  // threads per CTA = pixels per tile = floats per activation row

// Neuron groups of a hidden layer of width n: thread (pg, ng) owns TP = NG
// pixels and TN = n / NG neurons (NG x TN = n, 128 / NG pixel groups).
__host__ __device__ constexpr int ng_for(int n) { return n >= 64 ? 8 : (n >= 16 ? 4 : 2); }

// One hidden layer: K inputs, N outputs.  Shared-memory image: K weight rows
// then the bias row, each row holding, per 4-float chunk c and neuron group
// ng, neurons ng*TN + 4c .. 4c+3 (zero past TN): [row][c][ng][4].  A warp's
// load of chunk c is 32 (or fewer) consecutive words.
template <int K_, int N_>
struct Dense {
  static constexpr int K = K_, N = N_;
  static constexpr int NG = ng_for(N_), TN = N_ / NG, TP = NG, TN2 = TN / 2;
  static constexpr int NCH = (TN + 3) / 4;
  static constexpr int ROWF = NCH * NG * 4;
  static constexpr int FLOATS = (K + 1) * ROWF;
  static_assert(N_ % NG == 0 && TN % 2 == 0, "hidden width must split into even neuron groups");
};

// Copies one hidden layer from the nn.Linear layout (W [N][K] row-major,
// then b [N]) into its shared-memory image.
template <class Ly>
__device__ __forceinline__ void load_dense(float* __restrict__ sm, const float* __restrict__ w) {
  for (int e = threadIdx.x; e < Ly::FLOATS; e += kThreads) {
    const int k = e / Ly::ROWF, r = e - k * Ly::ROWF;
    const int c = r / (4 * Ly::NG), r2 = r - c * 4 * Ly::NG;
    const int ng = r2 >> 2, j = 4 * c + (r2 & 3);
    const int n = ng * Ly::TN + j;
    float v = 0.0f;
    if (j < Ly::TN) v = k < Ly::K ? w[n * Ly::K + k] : w[Ly::N * Ly::K + n];
    sm[e] = v;
  }
}

// The output layer (K inputs, 3 outputs): rows [k][4] = W[0..2][k], 0, then
// the bias row.
template <int K>
__device__ __forceinline__ void load_out(float* __restrict__ sm, const float* __restrict__ w) {
  for (int e = threadIdx.x; e < (K + 1) * 4; e += kThreads) {
    const int k = e >> 2, c = e & 3;
    float v = 0.0f;
    if (c < 3) v = k < K ? w[c * K + k] : w[3 * K + c];
    sm[e] = v;
  }
}

// The TP activations of pixel group pg in a 128-float row whose 16-byte
// chunks are XOR-swizzled by sw: TP = 8 -> chunks 2pg, 2pg+1; TP = 4 ->
// chunk pg; TP = 2 -> half of chunk pg / 2.
template <int TP>
__device__ __forceinline__ void load_px(const float* __restrict__ row, int pg, int sw, float (&a)[TP]) {
  if constexpr (TP == 8) {
    const float4 u = *reinterpret_cast<const float4*>(row + (((2 * pg) ^ sw) << 2));
    const float4 v = *reinterpret_cast<const float4*>(row + (((2 * pg + 1) ^ sw) << 2));
    a[0] = u.x; a[1] = u.y; a[2] = u.z; a[3] = u.w;
    a[4] = v.x; a[5] = v.y; a[6] = v.z; a[7] = v.w;
  } else if constexpr (TP == 4) {
    const float4 u = *reinterpret_cast<const float4*>(row + ((pg ^ sw) << 2));
    a[0] = u.x; a[1] = u.y; a[2] = u.z; a[3] = u.w;
  } else {
    static_assert(TP == 2, "pixels per thread: 2, 4 or 8");
    const float2 u = *reinterpret_cast<const float2*>(row + (((pg >> 1) ^ sw) << 2) + ((pg & 1) << 1));
    a[0] = u.x; a[1] = u.y;
  }
}

template <int TP>
__device__ __forceinline__ void store_px(float* __restrict__ row, int pg, int sw, const float (&a)[TP]) {
  if constexpr (TP == 8) {
    *reinterpret_cast<float4*>(row + (((2 * pg) ^ sw) << 2)) = make_float4(a[0], a[1], a[2], a[3]);
    *reinterpret_cast<float4*>(row + (((2 * pg + 1) ^ sw) << 2)) = make_float4(a[4], a[5], a[6], a[7]);
  } else if constexpr (TP == 4) {
    *reinterpret_cast<float4*>(row + ((pg ^ sw) << 2)) = make_float4(a[0], a[1], a[2], a[3]);
  } else {
    *reinterpret_cast<float2*>(row + (((pg >> 1) ^ sw) << 2) + ((pg & 1) << 1)) = make_float2(a[0], a[1]);
  }
}

// Float offset of pixel p in a row swizzled by sw.
__device__ __forceinline__ int px_off(int p, int sw) { return (((p >> 2) ^ sw) << 2) | (p & 3); }

// acc = b + X^T W over the layer's K input rows X[0 .. K) (row k swizzled by
// (k / BLK) & 7, or not at all when SWZ is false), for the thread's TP pixels
// and TN neurons; acc[p][j] packs neurons 2j, 2j+1 of pixel p.
template <class Ly, int BLK, bool SWZ>
__device__ __forceinline__ void dense_acc(const float* __restrict__ X, const float* __restrict__ Wl,
                                          int pg, int ng,
                                          unsigned long long (&acc)[Ly::TP][Ly::TN2]) {
  constexpr int TP = Ly::TP, TN2 = Ly::TN2, NCH = Ly::NCH, NG = Ly::NG, ROWF = Ly::ROWF;
  static_assert(Ly::K % BLK == 0, "input blocks must tile K");
  {
    const float* bias = Wl + Ly::K * ROWF + 4 * ng;
#pragma unroll
    for (int c = 0; c < NCH; ++c) {
      const ulonglong2 b = *reinterpret_cast<const ulonglong2*>(bias + c * 4 * NG);
#pragma unroll
      for (int p = 0; p < TP; ++p) {
        if (2 * c < TN2) acc[p][2 * c] = b.x;
        if (2 * c + 1 < TN2) acc[p][2 * c + 1] = b.y;
      }
    }
  }
#pragma unroll 2
  for (int kb = 0; kb < Ly::K / BLK; ++kb) {
    const int sw = SWZ ? (kb & 7) : 0;
    const float* xb = X + kb * BLK * kThreads;
    const float* wb = Wl + kb * BLK * ROWF + 4 * ng;
#pragma unroll
    for (int kk = 0; kk < BLK; ++kk) {
      float a[TP];
      load_px<TP>(xb + kk * kThreads, pg, sw, a);
      unsigned long long w[2 * NCH];
#pragma unroll
      for (int c = 0; c < NCH; ++c) {
        const ulonglong2 v = *reinterpret_cast<const ulonglong2*>(wb + kk * ROWF + c * 4 * NG);
        w[2 * c] = v.x;
        w[2 * c + 1] = v.y;
      }
#pragma unroll
      for (int p = 0; p < TP; ++p) {
        const unsigned long long ad = pack2(a[p], a[p]);
#pragma unroll
        for (int j = 0; j < TN2; ++j) acc[p][j] = fma2(ad, w[j], acc[p][j]);
      }
    }
  }
}

// The activation on every accumulator pair.
template <class Ly, int ACT>
__device__ __forceinline__ void activate_acc(unsigned long long (&acc)[Ly::TP][Ly::TN2]) {
#pragma unroll
  for (int p = 0; p < Ly::TP; ++p)
#pragma unroll
    for (int j = 0; j < Ly::TN2; ++j) {
      if constexpr (ACT == ACT_GELU) {
        acc[p][j] = gelu_poly2(acc[p][j]);
      } else {
        const float2 v = unpack2(acc[p][j]);
        acc[p][j] = pack2(fmaxf(v.x, 0.0f), fmaxf(v.y, 0.0f));
      }
    }
}

__device__ __forceinline__ float half_of(unsigned long long v, int hi) {
  const float2 f = unpack2(v);
  return hi ? f.y : f.x;
}

// Hidden-layer output: neuron ng*TN + j of the thread's pixels goes to row
// ng*TN + j of X, swizzled by ng & 7 (= (row / TN) & 7).
template <class Ly>
__device__ __forceinline__ void store_hidden(float* __restrict__ X, int pg, int ng,
                                             const unsigned long long (&acc)[Ly::TP][Ly::TN2]) {
  const int sw = ng & 7;
#pragma unroll
  for (int j = 0; j < Ly::TN; ++j) {
    float v[Ly::TP];
#pragma unroll
    for (int p = 0; p < Ly::TP; ++p) v[p] = half_of(acc[p][j >> 1], j & 1);
    store_px<Ly::TP>(X + (ng * Ly::TN + j) * kThreads, pg, sw, v);
  }
}

// Output-layer partial sums of the thread's TN neurons for its TP pixels:
// row 3 ng + c of X holds output c's partial from group ng, swizzled by
// ng & 7 (= (row / 3) & 7).
template <class Ly>
__device__ __forceinline__ void store_out_partials(float* __restrict__ X, const float* __restrict__ Wout,
                                                   int pg, int ng,
                                                   const unsigned long long (&acc)[Ly::TP][Ly::TN2]) {
  float part[3][Ly::TP];
#pragma unroll
  for (int c = 0; c < 3; ++c)
#pragma unroll
    for (int p = 0; p < Ly::TP; ++p) part[c][p] = 0.0f;
#pragma unroll
  for (int j = 0; j < Ly::TN; ++j) {
    const float4 w = *reinterpret_cast<const float4*>(Wout + 4 * (ng * Ly::TN + j));
#pragma unroll
    for (int p = 0; p < Ly::TP; ++p) {
      const float h = half_of(acc[p][j >> 1], j & 1);
      part[0][p] = fmaf(h, w.x, part[0][p]);
      part[1][p] = fmaf(h, w.y, part[1][p]);
      part[2][p] = fmaf(h, w.z, part[2][p]);
    }
  }
  const int sw = ng & 7;
#pragma unroll
  for (int c = 0; c < 3; ++c) store_px<Ly::TP>(X + (3 * ng + c) * kThreads, pg, sw, part[c]);
}

template <int C, int NL, int D0, int D1, int D2, int D3, int D4, int ACT>
struct Fp32Net {
  static_assert(NL >= 2 && NL <= 4, "1 to 3 hidden layers");
  static constexpr int L = D0 / C;
  using H1 = Dense<D0, D1>;
  using H2 = Dense<D1, (NL >= 3 ? D2 : 4)>;  // used only when NL >= 3
  using H3 = Dense<D2, (NL >= 4 ? D3 : 4)>;  // used only when NL >= 4
  static constexpr int KOUT = NL == 2 ? D1 : (NL == 3 ? D2 : D3);  // width of the last hidden layer
  static constexpr int NG_LAST = ng_for(KOUT);
  static constexpr int HMAX = (D1 > D2 ? D1 : D2) > D3 ? (D1 > D2 ? D1 : D2) : D3;
  // Rows of X: hidden outputs use [0, width); the output partials
  // [0, 3 NG_LAST); the features [F0, F0 + D0), clear of the partials so
  // that the next tile's features need no barrier after the RGB pass.
  static constexpr int F0 = (3 * NG_LAST > HMAX - D0) ? 3 * NG_LAST : HMAX - D0;
  static constexpr int XROWS = F0 + D0;
  static constexpr int OFF_H2 = H1::FLOATS;
  static constexpr int OFF_H3 = OFF_H2 + (NL >= 3 ? H2::FLOATS : 0);
  static constexpr int OFF_OUT = OFF_H3 + (NL >= 4 ? H3::FLOATS : 0);
  static constexpr int W_FLOATS = OFF_OUT + (KOUT + 1) * 4;
  static constexpr int smem_floats() { return W_FLOATS + XROWS * kThreads; }
  // CTAs per SM the shared memory allows (228 KB per SM, 1 KB reserved per
  // CTA), at most 4: the register budget per thread follows from it.
  static constexpr int MINB_RAW = (228 * 1024) / (smem_floats() * 4 + 1024);
  static constexpr int MINB = MINB_RAW < 1 ? 1 : (MINB_RAW > 4 ? 4 : MINB_RAW);
};

template <int C, int NL, int D0, int D1, int D2, int D3, int D4, int ACT, bool FL>
__global__ void __launch_bounds__(kThreads, (Fp32Net<C, NL, D0, D1, D2, D3, D4, ACT>::MINB))
    fp32_decode_kernel(const DecodeParams p) {
  using Net = Fp32Net<C, NL, D0, D1, D2, D3, D4, ACT>;
  using H1 = typename Net::H1;
  using H2 = typename Net::H2;
  using H3 = typename Net::H3;
  constexpr int L = Net::L;
  extern __shared__ __align__(16) float smem[];
  float* const sm_w = smem;
  float* const X = smem + Net::W_FLOATS;
  const float* const Wout = sm_w + Net::OFF_OUT;

  const int tid = threadIdx.x;
  const long long chunk = (p.total_tiles + gridDim.x - 1) / gridDim.x;
  const long long t_begin = blockIdx.x * chunk;
  const long long t_end = min(t_begin + chunk, p.total_tiles);
  const float* wts = static_cast<const float*>(p.weights);
  const long long plane = static_cast<long long>(p.H) * p.W;
  int cur_b = -1;

  for (long long t = t_begin; t < t_end; ++t) {
    const int b = static_cast<int>(t / p.tiles_per_image);
    const long long r = t - static_cast<long long>(b) * p.tiles_per_image;
    const int y = static_cast<int>(r / p.tiles_per_row);
    const int x = static_cast<int>(r - static_cast<long long>(y) * p.tiles_per_row) * kThreads + tid;
    if (b != cur_b) {  // uniform across the CTA
      __syncthreads();
      const float* w = wts + b * p.params_per_image;
      load_dense<H1>(sm_w, w);
      w += D1 * D0 + D1;
      if constexpr (NL >= 3) {
        load_dense<H2>(sm_w + Net::OFF_H2, w);
        w += D2 * D1 + D2;
      }
      if constexpr (NL >= 4) {
        load_dense<H3>(sm_w + Net::OFF_H3, w);
        w += D3 * D2 + D3;
      }
      load_out<Net::KOUT>(sm_w + Net::OFF_OUT, w);
      cur_b = b;
      __syncthreads();
    }

    // ---- steps 1-3: dequantise, upsample and concatenate every level ----
    // (pixels past the row's end decode column W - 1 and are not stored)
    {
      const int xc = min(x, p.W - 1);
      const int32_t* lat = p.latents + b * p.lat_per_image;
      float* f = X + Net::F0 * kThreads + tid;
#pragma unroll
      for (int l = 0; l < L; ++l) {
        const LevelGeom lg = p.lv[l];
        const float step = FL ? 1.0f : __ldg(p.steps + b * L + l);  // uniform: one broadcast load
        if (l == 0) {  // level 0 has the output size: the upsampling is the identity
#pragma unroll
          for (int c = 0; c < C; ++c)
            f[c * kThreads] =
                step * lat_value<FL>(__ldg(lat + c * plane + static_cast<long long>(y) * p.W + xc));
        } else {
          const Tap tx = bilinear_tap(xc, lg.sx, lg.W);
          const Tap ty = bilinear_tap(y, lg.sy, lg.H);
#pragma unroll
          for (int c = 0; c < C; ++c)
            f[(l * C + c) * kThreads] =
                step * bilinear_sample<FL>(lat + lg.off + static_cast<long long>(c) * lg.H * lg.W,
                                           lg.W, tx, ty);
        }
      }
    }
    __syncthreads();

    // ---- step 4: the synthesis MLP ----
    {
      unsigned long long acc[H1::TP][H1::TN2];
      dense_acc<H1, D0, false>(X + Net::F0 * kThreads, sm_w, tid / H1::NG, tid % H1::NG, acc);
      activate_acc<H1, ACT>(acc);
      __syncthreads();
      if constexpr (NL == 2)
        store_out_partials<H1>(X, Wout, tid / H1::NG, tid % H1::NG, acc);
      else
        store_hidden<H1>(X, tid / H1::NG, tid % H1::NG, acc);
      __syncthreads();
    }
    if constexpr (NL >= 3) {
      unsigned long long acc[H2::TP][H2::TN2];
      dense_acc<H2, H1::TN, true>(X, sm_w + Net::OFF_H2, tid / H2::NG, tid % H2::NG, acc);
      activate_acc<H2, ACT>(acc);
      __syncthreads();
      if constexpr (NL == 3)
        store_out_partials<H2>(X, Wout, tid / H2::NG, tid % H2::NG, acc);
      else
        store_hidden<H2>(X, tid / H2::NG, tid % H2::NG, acc);
      __syncthreads();
    }
    if constexpr (NL >= 4) {
      unsigned long long acc[H3::TP][H3::TN2];
      dense_acc<H3, H2::TN, true>(X, sm_w + Net::OFF_H3, tid / H3::NG, tid % H3::NG, acc);
      activate_acc<H3, ACT>(acc);
      __syncthreads();
      store_out_partials<H3>(X, Wout, tid / H3::NG, tid % H3::NG, acc);
      __syncthreads();
    }

    // ---- output layer sums and step 5: clamp and store ----
    if (x < p.W) {
      const float* bo = Wout + Net::KOUT * 4;
      float o0 = bo[0], o1 = bo[1], o2 = bo[2];
#pragma unroll
      for (int g = 0; g < Net::NG_LAST; ++g) {
        const int off = px_off(tid, g & 7);
        o0 += X[(3 * g) * kThreads + off];
        o1 += X[(3 * g + 1) * kThreads + off];
        o2 += X[(3 * g + 2) * kThreads + off];
      }
      store_rgb(p, b, y, x, o0, o1, o2);
    }
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
