// pic_common.cuh -- launch parameters and device helpers shared by the decode
// kernels (the CUDA path only; the fp64 oracle shares nothing with this file).
#pragma once

#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>
#include <cuda_fp16.h>

#include "pic_gelu.cuh"

namespace pic {

constexpr int kMaxLevels = 12;
constexpr int kMaxLayers = 6;
constexpr int kMaxDim = 128;

// Tensor-core tiles: 128 pixels of one image row (one tensor-memory lane
// each).  The TMA-staged kernels load a tile's full-resolution row segment
// (level 0) of each channel as one TMA box of kTmaRowBox 4-byte words: the
// box starts at the segment's first word rounded down to a multiple of 4
// (TMA's 16-byte rule), so 3 more words than the tile's 128 and a multiple
// of 4 in all.
constexpr int kTcTile = 128;
constexpr int kTmaRowBox = kTcTile + 4;

// Geometry of one pyramid level (Eq. 1 with the ceiling rule): size, offset
// of the level inside one image's latent block, and the size ratios
// W_l / W, H_l / H that map output pixel centres to source coordinates.
struct LevelGeom {
  int H, W;
  long long off;   // element offset of level l within one image's latents
  float sx, sy;    // W_l / W and H_l / H, rounded to fp32
};

// Everything a decode launch needs; passed by value (kernel parameter space).
struct DecodeParams {
  const int32_t* latents;      // int32 symbols, or fp32 values (PIC_LATENT_FP32) as 32-bit words
  const float* steps;
  const void* weights;
  void* out;                   // fp32 [B][3][H][W], fp32 [B][H][W][3] or uint8 [B][H][W][3]
  int H, W, B, L, C;
  int clamp;
  int out_format;              // OUT_F32_CHW, OUT_F32_HWC or OUT_U8_HWC
  long long lat_per_image;     // sum_l C H_l W_l
  long long params_per_image;  // sum_k d_{k+1} (d_k + 1)
  int tiles_per_row;
  long long tiles_per_image;
  long long total_tiles;
  int* status;                 // device word: nonzero after a bounded wait gave up
  int n_layers;
  int dims[kMaxLayers + 1];
  int act;
  LevelGeom lv[kMaxLevels];
  unsigned spin_limit;         // polls a bounded device-side wait makes before giving up
  int test_fault;              // tests of the bounded waits only (0 in production)
};

// Polls a bounded device-side wait makes before it gives up (with a short
// sleep between polls after the first few thousand): seconds at most.
constexpr unsigned kWaitPolls = 1u << 22;

// Tensor map for the TMA staging of the tensor-core kernels: the whole
// latent buffer of the call (every image's pyramid) as one 1-D tensor of
// 4-byte words with boxes of kTmaRowBox words; a box reads zeros past the
// buffer's end.
struct TmaParams {
  CUtensorMap lat;
};

enum { ACT_RELU = 0, ACT_GELU = 1 };
enum { OUT_F32_CHW = 0, OUT_F32_HWC = 1, OUT_U8_HWC = 2 };

// Step 5 for pixel (x, y) of image b: clamp (unless the handle asks for raw
// values) and store in the handle's output format.  uint8 is
// round-half-even(255 clamp(v, 0, 1)) and always clamps.
__device__ __forceinline__ void store_rgb(const DecodeParams& p, int b, int y, int x, float r, float g,
                                          float bl) {
  const long long plane = static_cast<long long>(p.H) * p.W;
  const long long pix = static_cast<long long>(y) * p.W + x;
  if (p.out_format == OUT_U8_HWC) {
    uint8_t* o = static_cast<uint8_t*>(p.out) + (static_cast<long long>(b) * plane + pix) * 3;
    o[0] = static_cast<uint8_t>(__float2int_rn(__saturatef(r) * 255.0f));
    o[1] = static_cast<uint8_t>(__float2int_rn(__saturatef(g) * 255.0f));
    o[2] = static_cast<uint8_t>(__float2int_rn(__saturatef(bl) * 255.0f));
    return;
  }
  if (p.clamp) {
    r = __saturatef(r);
    g = __saturatef(g);
    bl = __saturatef(bl);
  }
  if (p.out_format == OUT_F32_HWC) {
    float* o = static_cast<float*>(p.out) + (static_cast<long long>(b) * plane + pix) * 3;
    o[0] = r;
    o[1] = g;
    o[2] = bl;
  } else {
    float* o = static_cast<float*>(p.out) + static_cast<long long>(b) * 3 * plane + pix;
    o[0] = r;
    o[plane] = g;
    o[2 * plane] = bl;
  }
}

// GELU in its erf form, z * Phi(z), with CUDA's erff (reference variant).
__device__ __forceinline__ float gelu_erf(float z) {
  return 0.5f * z * (1.0f + erff(z * 0.70710678118654752f));
}

// ---- packed fp32 pairs (sm_100+ f32x2 instructions) ----------------------
__device__ __forceinline__ unsigned long long pack2(float lo, float hi) {
  unsigned long long r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ float2 unpack2(unsigned long long v) {
  float2 r;
  asm("mov.b64 {%0, %1}, %2;" : "=f"(r.x), "=f"(r.y) : "l"(v));
  return r;
}
// d = a * b + c on both halves (one instruction, two FMAs).
__device__ __forceinline__ unsigned long long fma2(unsigned long long a, unsigned long long b,
                                                   unsigned long long c) {
  unsigned long long d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}

// d = a - b on both halves.
__device__ __forceinline__ unsigned long long sub2(unsigned long long a, unsigned long long b) {
  unsigned long long d;
  asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}

// d = a * b on both halves.
__device__ __forceinline__ unsigned long long mul2(unsigned long long a, unsigned long long b) {
  unsigned long long d;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}

// 1 / x on the special-function unit (rcp.approx: within an ulp; x >= 1
// wherever the GELU uses it).
__device__ __forceinline__ float rcp_approx(float x) {
  float r;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}

// GELU z * Phi(z) without branches (the rational function of gen_gelu.py,
// max abs error ~1.2e-6 in fp32):
//   s = min(z^2, Z^2), Phi = saturate(1/2 + z P(s) / Q(s)),
// the saturation being both the clamp Phi in [0, 1] and the value beyond Z.
// 13 FP32-pipe operations and one reciprocal per value.
__device__ __forceinline__ float gelu_approx(float z) {
  const float s = fminf(z * z, kGeluZ2);
  float pn = gelu_p(0), qd = gelu_q(0);
#pragma unroll
  for (int i = 1; i <= kGeluDegP; ++i) pn = fmaf(pn, s, gelu_p(i));
#pragma unroll
  for (int i = 1; i <= kGeluDegQ; ++i) qd = fmaf(qd, s, gelu_q(i));
  return z * __saturatef(fmaf(z, pn * rcp_approx(qd), 0.5f));
}

// The same on a pair of values packed in 64 bits: the multiplies and the
// Horner chains run as packed f32x2 instructions (one instruction, two
// operations), with the same roundings as gelu_approx on each half.
__device__ __forceinline__ unsigned long long gelu_approx2(unsigned long long v) {
  const float2 zz = unpack2(mul2(v, v));
  const unsigned long long s = pack2(fminf(zz.x, kGeluZ2), fminf(zz.y, kGeluZ2));
  unsigned long long pn = pack2(gelu_p(0), gelu_p(0)), qd = pack2(gelu_q(0), gelu_q(0));
#pragma unroll
  for (int i = 1; i <= kGeluDegP; ++i) pn = fma2(pn, s, pack2(gelu_p(i), gelu_p(i)));
#pragma unroll
  for (int i = 1; i <= kGeluDegQ; ++i) qd = fma2(qd, s, pack2(gelu_q(i), gelu_q(i)));
  const float2 q = unpack2(qd);
  const float2 r = unpack2(mul2(pn, pack2(rcp_approx(q.x), rcp_approx(q.y))));
  const float2 z = unpack2(v);
  return mul2(v, pack2(__saturatef(fmaf(z.x, r.x, 0.5f)), __saturatef(fmaf(z.y, r.y, 0.5f))));
}

template <int ACT>
__device__ __forceinline__ float activate(float z) {
  if constexpr (ACT == ACT_GELU) return gelu_approx(z);
  else return fmaxf(z, 0.0f);
}

__device__ __forceinline__ float activate_rt(float z, int act) {
  return act == ACT_GELU ? gelu_approx(z) : fmaxf(z, 0.0f);
}

// Bilinear source coordinate of output index x along one axis: the pixel
// centre x + 1/2 maps to (x + 1/2) * ratio - 1/2, clamped below at 0; i0 is
// its floor, i1 the next index clamped to n - 1, and frac the weight of i1.
struct Tap {
  int i0, i1;
  float frac;
};
__device__ __forceinline__ Tap bilinear_tap(int x, float ratio, int n) {
  float s = fmaxf(fmaf(static_cast<float>(x) + 0.5f, ratio, -0.5f), 0.0f);
  int i0 = static_cast<int>(s);
  Tap t;
  t.i0 = min(i0, n - 1);
  t.i1 = min(i0 + 1, n - 1);
  t.frac = s - static_cast<float>(i0);
  return t;
}

// Latent words: int32 symbols, or fp32 values carried in the same 32 bits
// (FL = true, PIC_LATENT_FP32).
template <bool FL>
__device__ __forceinline__ float lat_value(int w) {
  if constexpr (FL)
    return __int_as_float(w);
  else
    return static_cast<float>(w);
}
// a + t (b - a); for symbols the difference b - a is exact in integers.
template <bool FL>
__device__ __forceinline__ float lat_lerp(int a, int b, float t) {
  if constexpr (FL) {
    const float fa = __int_as_float(a);
    return fmaf(t, __int_as_float(b) - fa, fa);
  } else {
    return fmaf(t, static_cast<float>(b - a), static_cast<float>(a));
  }
}

// One bilinear sample of latent grid `q` (row stride w), in fp32: two
// horizontal lerps, then one vertical lerp.
template <bool FL>
__device__ __forceinline__ float bilinear_sample(const int32_t* __restrict__ q, int w, Tap tx,
                                                 Tap ty) {
  const int32_t* r0 = q + static_cast<long long>(ty.i0) * w;
  const int32_t* r1 = q + static_cast<long long>(ty.i1) * w;
  int a = __ldg(r0 + tx.i0), b = __ldg(r0 + tx.i1);
  int c = __ldg(r1 + tx.i0), d = __ldg(r1 + tx.i1);
  float top = lat_lerp<FL>(a, b, tx.frac);
  float bot = lat_lerp<FL>(c, d, tx.frac);
  return fmaf(ty.frac, bot - top, top);
}

}  // namespace pic
