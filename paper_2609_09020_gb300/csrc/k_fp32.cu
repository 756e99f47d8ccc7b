// k_fp32.cu -- instantiations of the fp32 CUDA-core decode kernel
// (k_fp32.cuh) for the decode workloads' architectures, the generic
// kernel and the registry of all fp32 kernels.
#include "k_fp32.cuh"

namespace pic {

// Instantiations: the decode workloads' architectures, specialised at compile
// time; anything else runs on the generic kernel.
int fp32_kernels(KernelInfo* out, int cap) {
  const KernelInfo list[] = {
      make_fp32<1, 3, 4, 16, 16, 3, 0, ACT_RELU>("fp32_4x16x16x3_relu"),
      make_fp32<1, 3, 7, 40, 40, 3, 0, ACT_GELU>("fp32_7x40x40x3_gelu"),
      make_fp32<2, 3, 14, 64, 64, 3, 0, ACT_RELU>("fp32_14x64x64x3_relu"),
      make_fp32<2, 4, 16, 64, 64, 64, 3, ACT_GELU>("fp32_16x64x64x64x3_gelu"),
      make_fp32<1, 3, 7, 64, 64, 3, 0, ACT_RELU>("fp32_7x64x64x3_relu"),
      make_fp32<1, 3, 7, 64, 64, 3, 0, ACT_RELU, true>("fp32_7x64x64x3_relu_f32lat"),
  };
  const int n = static_cast<int>(sizeof(list) / sizeof(list[0]));
  int k = 0;
  for (; k < n && k < cap; ++k) out[k] = list[k];
  if (k < cap) k += fp32_kernels_sweep(out + k, cap - k);
  return k;
}

KernelInfo fp32_generic_kernel_info(int latent_format) {
  KernelInfo k{};
  k.name = latent_format ? "fp32_generic_f32lat" : "fp32_generic";
  k.precision = 0;
  k.latent_format = latent_format ? 1 : 0;
  k.generic = 1;
  k.threads = kThreads;
  k.tile_px = kThreads;
  k.smem_bytes = 0;  // set per arch: params_per_image * 4
  k.fn = latent_format ? reinterpret_cast<const void*>(&fp32_generic_kernel<true>)
                      : reinterpret_cast<const void*>(&fp32_generic_kernel<false>);
  return k;
}

}  // namespace pic
