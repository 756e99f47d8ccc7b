// k_fuse.cu -- modulation fusion (include/pic_fuse.h; Sec. 3.1 Eqs. 2-3,
// App. A).  One CTA per image: the threads copy the shared layers (and
// convert them to the output dtype), scale the last layer's columns by
// gamma_c / sigma_c, and one warp per output row reduces
// b[i] + sum_c w[i][c] (beta_c - gamma_c mu_c / sigma_c) with shuffles.
#include <cstdint>

#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "pic_decode.h"
#include "pic_fuse.h"

namespace {

constexpr int kThreads = 256;
constexpr int kMaxLayers = 6;

struct FuseParams {
  const float* shared;
  const float* mod;
  void* out;
  long long P;       // weights per image
  long long last;    // offset of the last layer's W in the blob
  int dout, cf;      // last layer: dout rows of cf inputs
  int half;          // 1: IEEE half output
};

template <bool HALF>
__device__ __forceinline__ void put(void* out, long long i, float v) {
  if constexpr (HALF)
    static_cast<__half*>(out)[i] = __float2half_rn(v);
  else
    static_cast<float*>(out)[i] = v;
}

template <bool HALF>
__global__ void __launch_bounds__(kThreads) fuse_kernel(const FuseParams p) {
  const int b = blockIdx.x;
  const float* gamma = p.mod + static_cast<long long>(b) * 4 * p.cf;
  const float* beta = gamma + p.cf;
  const float* mu = beta + p.cf;
  const float* sigma = mu + p.cf;
  const long long base = static_cast<long long>(b) * p.P;
  const long long wend = p.last + static_cast<long long>(p.dout) * p.cf;  // last layer's bias starts here
  for (long long e = threadIdx.x; e < p.P; e += kThreads) {
    float v = __ldg(p.shared + e);
    if (e >= p.last && e < wend) {
      const int c = static_cast<int>((e - p.last) % p.cf);
      v = v * __ldg(gamma + c) / __ldg(sigma + c);
    }
    if (e < p.last || e < wend) put<HALF>(p.out, base + e, v);
  }
  // fused biases: warp i reduces row i
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int i = warp; i < p.dout; i += kThreads / 32) {
    const float* w = p.shared + p.last + static_cast<long long>(i) * p.cf;
    float s = 0.0f;
    for (int c = lane; c < p.cf; c += 32)
      s = fmaf(__ldg(w + c), __ldg(beta + c) - __ldg(gamma + c) * __ldg(mu + c) / __ldg(sigma + c), s);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if (lane == 0) put<HALF>(p.out, base + wend + i, __ldg(p.shared + wend + i) + s);
  }
}

}  // namespace

extern "C" int pic_fuse_modulation(const pic_arch* arch, int B, const float* shared,
                                   const float* mod, void* weights_out, void* stream) {
  if (!arch || !shared || !mod || !weights_out || B < 1 || B > 65536) return PIC_ERR_INVALID_ARG;
  const int n = arch->num_layers;
  if (n < 2 || n > kMaxLayers) return PIC_ERR_INVALID_ARG;
  long long P = 0, last = 0;
  for (int k = 0; k < n; ++k) {
    if (arch->dims[k] < 1 || arch->dims[k + 1] < 1 || arch->dims[k] > 128 || arch->dims[k + 1] > 128)
      return PIC_ERR_INVALID_ARG;
    if (k == n - 1) last = P;
    P += static_cast<long long>(arch->dims[k + 1]) * (arch->dims[k] + 1);
  }
  const bool half = arch->precision == PIC_PREC_FP16_TC || arch->precision == PIC_PREC_FP16_TC_LO8;
  if (!half && arch->precision != PIC_PREC_FP32) return PIC_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(weights_out) & 15u) != 0 ||
      (reinterpret_cast<uintptr_t>(shared) & 3u) != 0 || (reinterpret_cast<uintptr_t>(mod) & 3u) != 0)
    return PIC_ERR_INVALID_ARG;
  FuseParams p{shared, mod, weights_out, P, last, arch->dims[n], arch->dims[n - 1], half ? 1 : 0};
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (half)
    fuse_kernel<true><<<B, kThreads, 0, s>>>(p);
  else
    fuse_kernel<false><<<B, kThreads, 0, s>>>(p);
  if (cudaGetLastError() != cudaSuccess) return PIC_ERR_CUDA;
  return PIC_OK;
}
