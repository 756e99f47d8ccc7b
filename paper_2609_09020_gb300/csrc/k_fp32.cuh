// k_fp32.cuh -- the fp32 CUDA-core decode kernel templates (PIC_PREC_FP32),
// instantiated in k_fp32.cu (the decode workloads' architectures, the
// generic kernel, the registry) and k_fp32_sweep.cu (the width ablation).
//
// The decode fused on the fp32 CUDA cores, in two kernels: the
// register-tiled contraction below (nets with a hidden layer wider than 16)
// and, further down, one thread per pixel for narrower nets.
//
// Register-tiled: a CTA of 128 threads decodes tiles of 128 consecutive
// pixels of one image row.  Per tile:
//   1. features: thread p dequantises and upsamples every pyramid level for
//      pixel p (Sec. 3.1, Eq. 1) and writes the feature vector into a
//      shared-memory activation buffer X (one row of 128 floats per
//      feature), so features never reach HBM;
//   2. each hidden layer of g_s (Sec. 4.1) is a 128-pixel x N contraction
//      on the CUDA cores, register-tiled: warp ng owns the neurons
//      ng*TN .. ng*TN + TN - 1 (TN = N / 4) and its lane pg the 4 pixels
//      4pg .. 4pg + 3, and accumulates those 4 x TN outputs over the K
//      inputs.  Per input a lane loads its 4 activations (one 16-byte load;
//      a quarter-warp reads 128 consecutive bytes) and the warp's TN weights
//      (16-byte loads at one address for the whole warp, a broadcast), so
//      each load feeds TN (resp. 4) FMAs; packed f32x2 FMAs do two neurons of
//      one pixel per instruction.  The bias seeds the accumulators; the
//      activation is applied in registers and the layer's output rows are
//      written back over X (again 128 consecutive bytes per quarter-warp);
//   3. the output layer (3 neurons) is folded into the last hidden layer's
//      epilogue: each lane forms the 3 partial sums over its warp's TN
//      neurons for its 4 pixels, and thread p adds the 4 warps' partials of
//      pixel p and the bias, clamps and stores the planar RGB row
//      (coalesced).
// Weights live in shared memory for the whole tile range (reloaded when the
// image changes).
//
// Work split: the tiles of all images are numbered image-major and each CTA
// takes one contiguous range of them, all ranges within one tile of the same
// length (a CTA sees at most a couple of images and loads each one's weights
// once).  Grid = resident CTAs over all SMs.

#pragma once

#include "pic_common.cuh"
#include "pic_kernels.h"

namespace pic {
namespace {

constexpr int kThreads = 128;  // threads per CTA = pixels per tile = floats per activation row
constexpr int kWarps = kThreads / 32;  // neuron groups of a layer
constexpr int kTP = 4;                 // pixels per lane

// One hidden layer: K inputs, N outputs, warp ng computing neurons
// ng*TN .. ng*TN + TN - 1.  Shared-memory image: K weight rows then the bias
// row, each row holding per warp a segment of SEGF floats (its TN neurons,
// zero padded to whole 16-byte chunks): [row][ng][SEGF].
template <int K_, int N_>
struct Dense {
  static constexpr int K = K_, N = N_;
  static constexpr int TN = N_ / kWarps, TN2 = TN / 2;
  static constexpr int NCH = (TN + 3) / 4;
  static constexpr int SEGF = 4 * NCH;
  static constexpr int ROWF = kWarps * SEGF;
  static constexpr int FLOATS = (K + 1) * ROWF;
  // inputs per iteration of the K loop
  static constexpr int UNR = K <= 16 ? K : (K % 16 == 0 ? 16 : (K % 8 == 0 ? 8 : 1));
  static_assert(N_ % (2 * kWarps) == 0, "hidden width must be a multiple of 8");
};

// Copies one hidden layer from the nn.Linear layout (W [N][K] row-major,
// then b [N]) into its shared-memory image.
template <class Ly>
__device__ __forceinline__ void load_dense(float* __restrict__ sm, const float* __restrict__ w) {
  for (int e = threadIdx.x; e < Ly::FLOATS; e += kThreads) {
    const int k = e / Ly::ROWF, r = e - k * Ly::ROWF;
    const int ng = r / Ly::SEGF, j = r - ng * Ly::SEGF;
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

// acc = b + X^T W over the layer's K input rows X[0 .. K), for lane pg's 4
// pixels and warp ng's TN neurons; acc[p][j] packs neurons 2j, 2j+1 of
// pixel 4pg + p.
template <class Ly>
__device__ __forceinline__ void dense_acc(const float* __restrict__ X, const float* __restrict__ Wl,
                                          int pg, int ng, unsigned long long (&acc)[kTP][Ly::TN2]) {
  constexpr int TN2 = Ly::TN2, NCH = Ly::NCH, ROWF = Ly::ROWF;
  const float* wseg = Wl + ng * Ly::SEGF;  // warp-uniform
  {
    const float* bias = wseg + Ly::K * ROWF;
#pragma unroll
    for (int c = 0; c < NCH; ++c) {
      const ulonglong2 b = *reinterpret_cast<const ulonglong2*>(bias + 4 * c);
#pragma unroll
      for (int p = 0; p < kTP; ++p) {
        if (2 * c < TN2) acc[p][2 * c] = b.x;
        if (2 * c + 1 < TN2) acc[p][2 * c + 1] = b.y;
      }
    }
  }
  const float* xa = X + 4 * pg;
#pragma unroll 1
  for (int k0 = 0; k0 < Ly::K; k0 += Ly::UNR) {
#pragma unroll
    for (int kk = 0; kk < Ly::UNR; ++kk) {
      const float4 a = *reinterpret_cast<const float4*>(xa + (k0 + kk) * kThreads);
      unsigned long long w[2 * NCH];
#pragma unroll
      for (int c = 0; c < NCH; ++c) {
        const ulonglong2 v = *reinterpret_cast<const ulonglong2*>(wseg + (k0 + kk) * ROWF + 4 * c);
        w[2 * c] = v.x;
        w[2 * c + 1] = v.y;
      }
      const unsigned long long ad[kTP] = {pack2(a.x, a.x), pack2(a.y, a.y), pack2(a.z, a.z),
                                          pack2(a.w, a.w)};
#pragma unroll
      for (int p = 0; p < kTP; ++p)
#pragma unroll
        for (int j = 0; j < TN2; ++j) acc[p][j] = fma2(ad[p], w[j], acc[p][j]);
    }
  }
}

// The activation on every accumulator pair.
template <class Ly, int ACT>
__device__ __forceinline__ void activate_acc(unsigned long long (&acc)[kTP][Ly::TN2]) {
#pragma unroll
  for (int p = 0; p < kTP; ++p)
#pragma unroll
    for (int j = 0; j < Ly::TN2; ++j) {
      if constexpr (ACT == ACT_GELU) {
        acc[p][j] = gelu_approx2(acc[p][j]);
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

// Hidden-layer output: neuron ng*TN + j of lane pg's pixels goes to row
// ng*TN + j of X.
template <class Ly>
__device__ __forceinline__ void store_hidden(float* __restrict__ X, int pg, int ng,
                                             const unsigned long long (&acc)[kTP][Ly::TN2]) {
#pragma unroll
  for (int j = 0; j < Ly::TN; ++j) {
    float v[kTP];
#pragma unroll
    for (int p = 0; p < kTP; ++p) v[p] = half_of(acc[p][j >> 1], j & 1);
    *reinterpret_cast<float4*>(X + (ng * Ly::TN + j) * kThreads + 4 * pg) = make_float4(v[0], v[1], v[2], v[3]);
  }
}

// Output-layer partial sums of warp ng's TN neurons for lane pg's pixels:
// row 3 ng + c of X holds output c's partial from warp ng.
template <class Ly>
__device__ __forceinline__ void store_out_partials(float* __restrict__ X, const float* __restrict__ Wout,
                                                   int pg, int ng,
                                                   const unsigned long long (&acc)[kTP][Ly::TN2]) {
  float part[3][kTP];
#pragma unroll
  for (int c = 0; c < 3; ++c)
#pragma unroll
    for (int p = 0; p < kTP; ++p) part[c][p] = 0.0f;
#pragma unroll
  for (int j = 0; j < Ly::TN; ++j) {
    const float4 w = *reinterpret_cast<const float4*>(Wout + 4 * (ng * Ly::TN + j));
#pragma unroll
    for (int p = 0; p < kTP; ++p) {
      const float h = half_of(acc[p][j >> 1], j & 1);
      part[0][p] = fmaf(h, w.x, part[0][p]);
      part[1][p] = fmaf(h, w.y, part[1][p]);
      part[2][p] = fmaf(h, w.z, part[2][p]);
    }
  }
#pragma unroll
  for (int c = 0; c < 3; ++c)
    *reinterpret_cast<float4*>(X + (3 * ng + c) * kThreads + 4 * pg) =
        make_float4(part[c][0], part[c][1], part[c][2], part[c][3]);
}

template <int C, int NL, int D0, int D1, int D2, int D3, int D4, int ACT>
struct Fp32Net {
  static_assert(NL >= 2 && NL <= 4, "1 to 3 hidden layers");
  static constexpr int L = D0 / C;
  using H1 = Dense<D0, D1>;
  using H2 = Dense<D1, (NL >= 3 ? D2 : 8)>;  // used only when NL >= 3
  using H3 = Dense<D2, (NL >= 4 ? D3 : 8)>;  // used only when NL >= 4
  static constexpr int KOUT = NL == 2 ? D1 : (NL == 3 ? D2 : D3);  // width of the last hidden layer
  static constexpr int HMAX = (D1 > D2 ? D1 : D2) > D3 ? (D1 > D2 ? D1 : D2) : D3;
  // Rows of X: hidden outputs use [0, width); the output partials
  // [0, 3 kWarps); the features [F0, F0 + D0), clear of the partials so
  // that the next tile's features need no barrier after the RGB pass.
  static constexpr int F0 = (3 * kWarps > HMAX - D0) ? 3 * kWarps : HMAX - D0;
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
  const int warp = tid >> 5, lane = tid & 31;
  // balanced contiguous ranges: every CTA gets floor or ceil of tiles / CTAs
  const long long t_begin = blockIdx.x * p.total_tiles / gridDim.x;
  const long long t_end = (blockIdx.x + 1LL) * p.total_tiles / gridDim.x;
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
      unsigned long long acc[kTP][H1::TN2];
      dense_acc<H1>(X + Net::F0 * kThreads, sm_w, lane, warp, acc);
      activate_acc<H1, ACT>(acc);
      __syncthreads();
      if constexpr (NL == 2)
        store_out_partials<H1>(X, Wout, lane, warp, acc);
      else
        store_hidden<H1>(X, lane, warp, acc);
      __syncthreads();
    }
    if constexpr (NL >= 3) {
      unsigned long long acc[kTP][H2::TN2];
      dense_acc<H2>(X, sm_w + Net::OFF_H2, lane, warp, acc);
      activate_acc<H2, ACT>(acc);
      __syncthreads();
      if constexpr (NL == 3)
        store_out_partials<H2>(X, Wout, lane, warp, acc);
      else
        store_hidden<H2>(X, lane, warp, acc);
      __syncthreads();
    }
    if constexpr (NL >= 4) {
      unsigned long long acc[kTP][H3::TN2];
      dense_acc<H3>(X, sm_w + Net::OFF_H3, lane, warp, acc);
      activate_acc<H3, ACT>(acc);
      __syncthreads();
      store_out_partials<H3>(X, Wout, lane, warp, acc);
      __syncthreads();
    }

    // ---- output layer sums and step 5: clamp and store ----
    if (x < p.W) {
      const float* bo = Wout + Net::KOUT * 4;
      float o0 = bo[0], o1 = bo[1], o2 = bo[2];
#pragma unroll
      for (int g = 0; g < kWarps; ++g) {
        o0 += X[(3 * g) * kThreads + tid];
        o1 += X[(3 * g + 1) * kThreads + tid];
        o2 += X[(3 * g + 2) * kThreads + tid];
      }
      store_rgb(p, b, y, x, o0, o1, o2);
    }
  }
}

// ---------------------------------------------------------------------------
// Narrow nets (every hidden layer at most 16 wide): one thread per pixel with
// the features and every activation in registers, no activation buffer and
// no barrier per tile.  A 16-wide layer is only 16 FMAs per input, so the
// tiled kernel's fixed per-tile work (staging, barriers, partial sums) would
// outweigh the contraction.  Weights sit transposed in shared memory and are
// read with broadcast 16-byte loads; packed f32x2 FMAs do two outputs per
// instruction.

__host__ __device__ constexpr int round4(int d) { return (d + 3) & ~3; }

// Shared-memory image of one layer: W^T [din][round4(dout)] then the bias
// [round4(dout)], zero padded.
__host__ __device__ constexpr int px_layer_floats(int din, int dout) { return (din + 1) * round4(dout); }

__device__ __forceinline__ void load_px_layer(float* __restrict__ sm, const float* __restrict__ w, int din,
                                              int dout) {
  const int d4 = round4(dout);
  for (int e = threadIdx.x; e < (din + 1) * d4; e += kThreads) {
    const int j = e / d4, i = e - j * d4;  // row j of W^T (j == din: the bias row), column i
    float v = 0.0f;
    if (i < dout) v = (j < din) ? w[i * din + j] : w[dout * din + i];
    sm[e] = v;
  }
}

// out = act(W in + b), or W in + b for the output layer.
template <int DIN, int DOUT, int ACT, bool LAST, int MAXW>
__device__ __forceinline__ void dense_px(const float* __restrict__ wt, const float (&in)[MAXW],
                                         float (&out)[MAXW]) {
  constexpr int D4 = round4(DOUT);
  unsigned long long acc[D4 / 2];
#pragma unroll
  for (int i = 0; i < D4 / 4; ++i) {
    const ulonglong2 b = *reinterpret_cast<const ulonglong2*>(wt + DIN * D4 + 4 * i);
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
    if constexpr (ACT == ACT_GELU && !LAST) acc[i] = gelu_approx2(acc[i]);
    const float2 v = unpack2(acc[i]);
    const bool relu = !LAST && ACT == ACT_RELU;
    if (2 * i < DOUT) out[2 * i] = relu ? fmaxf(v.x, 0.0f) : v.x;
    if (2 * i + 1 < DOUT) out[2 * i + 1] = relu ? fmaxf(v.y, 0.0f) : v.y;
  }
}

template <int C, int NL, int D0, int D1, int D2, int D3, int D4, int ACT>
struct PxNet {
  static constexpr int L = D0 / C;
  static constexpr int MW = (D0 > 16 ? D0 : 16);  // widest vector a thread holds
  static constexpr int OFF2 = px_layer_floats(D0, D1);
  static constexpr int OFF3 = OFF2 + px_layer_floats(D1, D2);
  static constexpr int OFF4 = OFF3 + (NL >= 3 ? px_layer_floats(D2, D3) : 0);
  static constexpr int smem_floats() { return OFF4 + (NL >= 4 ? px_layer_floats(D3, D4) : 0); }
};

template <int C, int NL, int D0, int D1, int D2, int D3, int D4, int ACT, bool FL>
__global__ void __launch_bounds__(kThreads) fp32_px_kernel(const DecodeParams p) {
  using Net = PxNet<C, NL, D0, D1, D2, D3, D4, ACT>;
  constexpr int L = Net::L;
  constexpr int MW = Net::MW;
  extern __shared__ __align__(16) float sm_w[];

  const long long t_begin = blockIdx.x * p.total_tiles / gridDim.x;
  const long long t_end = (blockIdx.x + 1LL) * p.total_tiles / gridDim.x;
  const float* wts = static_cast<const float*>(p.weights);
  const long long plane = static_cast<long long>(p.H) * p.W;
  int cur_b = -1;

  for (long long t = t_begin; t < t_end; ++t) {
    const int b = static_cast<int>(t / p.tiles_per_image);
    const long long r = t - static_cast<long long>(b) * p.tiles_per_image;
    const int y = static_cast<int>(r / p.tiles_per_row);
    const int x = static_cast<int>(r - static_cast<long long>(y) * p.tiles_per_row) * kThreads +
                  threadIdx.x;
    if (b != cur_b) {  // uniform across the CTA
      __syncthreads();
      const float* w = wts + b * p.params_per_image;
      load_px_layer(sm_w, w, D0, D1);
      w += D1 * D0 + D1;
      load_px_layer(sm_w + Net::OFF2, w, D1, D2);
      w += D2 * D1 + D2;
      if constexpr (NL >= 3) {
        load_px_layer(sm_w + Net::OFF3, w, D2, D3);
        w += D3 * D2 + D3;
      }
      if constexpr (NL >= 4) load_px_layer(sm_w + Net::OFF4, w, D3, D4);
      __syncthreads();
      cur_b = b;
    }
    if (x >= p.W) continue;

    // ---- steps 1-3: dequantise, upsample and concatenate every level ----
    const int32_t* lat = p.latents + b * p.lat_per_image;
    float h[MW], g[MW];
#pragma unroll
    for (int l = 0; l < L; ++l) {
      const LevelGeom lg = p.lv[l];
      const float step = FL ? 1.0f : __ldg(p.steps + b * L + l);
      if (l == 0) {  // level 0 has the output size: the upsampling is the identity
#pragma unroll
        for (int c = 0; c < C; ++c)
          h[c] = step * lat_value<FL>(__ldg(lat + c * plane + static_cast<long long>(y) * p.W + x));
      } else {
        const Tap tx = bilinear_tap(x, lg.sx, lg.W);
        const Tap ty = bilinear_tap(y, lg.sy, lg.H);
#pragma unroll
        for (int c = 0; c < C; ++c)
          h[l * C + c] = step * bilinear_sample<FL>(lat + lg.off + static_cast<long long>(c) * lg.H * lg.W,
                                                    lg.W, tx, ty);
      }
    }

    // ---- step 4: the synthesis MLP (ping-pong between h and g) ----
    dense_px<D0, D1, ACT, false>(sm_w, h, g);
    if constexpr (NL == 2) {
      dense_px<D1, D2, ACT, true>(sm_w + Net::OFF2, g, h);
    } else {
      dense_px<D1, D2, ACT, false>(sm_w + Net::OFF2, g, h);
      if constexpr (NL == 3) {
        dense_px<D2, D3, ACT, true>(sm_w + Net::OFF3, h, g);
        for (int c = 0; c < 3; ++c) h[c] = g[c];
      } else {
        dense_px<D2, D3, ACT, false>(sm_w + Net::OFF3, h, g);
        dense_px<D3, D4, ACT, true>(sm_w + Net::OFF4, g, h);
      }
    }

    // ---- step 5: clamp and store (planar rows are coalesced) ----
    store_rgb(p, b, y, x, h[0], h[1], h[2]);
  }
}

// ---------------------------------------------------------------------------
// Generic kernel: any dims up to kMaxDim, runtime loops, weights in shared
// memory in the nn.Linear layout.  Slower (hidden values in local memory) but
// covers every arch the C ABI accepts.
template <bool FL>
__global__ void __launch_bounds__(kThreads) fp32_generic_kernel(const DecodeParams p) {
  extern __shared__ __align__(16) float sm_w[];
  // balanced contiguous ranges: every CTA gets floor or ceil of tiles / CTAs
  const long long t_begin = blockIdx.x * p.total_tiles / gridDim.x;
  const long long t_end = (blockIdx.x + 1LL) * p.total_tiles / gridDim.x;
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
  constexpr bool narrow = Net::HMAX <= 16;  // the one-thread-per-pixel kernel
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
  if constexpr (narrow) {
    k.smem_bytes = PxNet<C, NL, D0, D1, D2, D3, D4, ACT>::smem_floats() * 4;
    k.fn = reinterpret_cast<const void*>(&fp32_px_kernel<C, NL, D0, D1, D2, D3, D4, ACT, FL>);
  } else {
    k.smem_bytes = Net::smem_floats() * 4;
    k.fn = reinterpret_cast<const void*>(&fp32_decode_kernel<C, NL, D0, D1, D2, D3, D4, ACT, FL>);
  }
  return k;
}

}  // namespace
}  // namespace pic
