// k_fp32_sweep.cu -- instantiations of the fp32 CUDA-core decode kernel
// (k_fp32.cuh) for the width ablation's architectures: 8 single-channel
// levels and a 4-layer MLP 8-w-w-w-3 with ReLU, w = 8, 16, 32, 64.
#include "k_fp32.cuh"

namespace pic {

int fp32_kernels_sweep(KernelInfo* out, int cap) {
  const KernelInfo list[] = {
      make_fp32<1, 4, 8, 8, 8, 8, 3, ACT_RELU>("fp32_8x8x8x8x3_relu"),
      make_fp32<1, 4, 8, 16, 16, 16, 3, ACT_RELU>("fp32_8x16x16x16x3_relu"),
      make_fp32<1, 4, 8, 32, 32, 32, 3, ACT_RELU>("fp32_8x32x32x32x3_relu"),
      make_fp32<1, 4, 8, 64, 64, 64, 3, ACT_RELU>("fp32_8x64x64x64x3_relu"),
  };
  const int n = static_cast<int>(sizeof(list) / sizeof(list[0]));
  int k = 0;
  for (; k < n && k < cap; ++k) out[k] = list[k];
  return k;
}

}  // namespace pic
