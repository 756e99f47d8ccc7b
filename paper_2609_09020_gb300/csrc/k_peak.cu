// k_peak.cu -- FP32 FMA throughput microbenchmark behind include/pic_measure.h:
// the peak of the CUDA cores that the fp32 decode path is measured against.
#include <cstdint>

#include <cuda_runtime.h>

#include "pic_decode.h"
#include "pic_measure.h"

namespace {

constexpr int kThreads = 256;
constexpr int kChains = 8;   // independent chains per thread: FMA latency hidden by ILP
constexpr int kUnroll = 16;  // FMAs per chain per iteration

__global__ void __launch_bounds__(kThreads) fma_peak_kernel(float* out, int iters, float a, float b) {
  float x[kChains];
#pragma unroll
  for (int k = 0; k < kChains; ++k) x[k] = static_cast<float>(threadIdx.x) * 1e-3f + static_cast<float>(k);
  for (int i = 0; i < iters; ++i) {
#pragma unroll
    for (int r = 0; r < kUnroll; ++r)
#pragma unroll
      for (int k = 0; k < kChains; ++k) x[k] = fmaf(x[k], a, b);
  }
  float s = 0.0f;
#pragma unroll
  for (int k = 0; k < kChains; ++k) s += x[k];
  if (s == -1.0f) out[blockIdx.x] = s;  // never true for the arguments passed; keeps the work
}

}  // namespace

extern "C" {

int64_t pic_fma_peak_flops(int blocks, int iters) {
  if (blocks < 1 || iters < 1) return -1;
  return static_cast<int64_t>(blocks) * kThreads * iters * kUnroll * kChains * 2;
}

int pic_fma_peak_launch(float* out, int blocks, int iters, void* stream) {
  if (!out || blocks < 1 || iters < 1) return PIC_ERR_INVALID_ARG;
  // x -> 0.999999 x + 1e-6 stays in [0, 1000) for these starting values
  fma_peak_kernel<<<blocks, kThreads, 0, static_cast<cudaStream_t>(stream)>>>(out, iters, 0.999999f, 1e-6f);
  if (cudaGetLastError() != cudaSuccess) return PIC_ERR_CUDA;
  return PIC_OK;
}

}  // extern "C"
