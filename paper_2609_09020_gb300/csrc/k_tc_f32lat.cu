// k_tc_f32lat.cu -- instantiations of the tensor-core decode kernel
// (k_tc.cuh) for fp32 latents (PIC_LATENT_FP32, the inverse DCT stage's
// output): the same architectures as the int32 set.
#include "k_tc.cuh"

namespace pic {
namespace {
const int d_c1[] = {4, 16, 16, 3};
const int d_c2[] = {7, 40, 40, 3};
const int d_c3[] = {14, 64, 64, 3};
const int d_c4[] = {16, 64, 64, 64, 3};
const int d_c5[] = {7, 64, 64, 3};
}  // namespace

int tc_kernels_fp32lat(KernelInfo* out, int cap) {
  const KernelInfo list[] = {
      make_tc<1, 3, 7, 64, ACT_RELU, 4, true>("tc05_7x64x64x3_relu_f32lat", d_c5),
      make_tc<2, 4, 16, 64, ACT_GELU, 4, true>("tc05_16x64x64x64x3_gelu_f32lat", d_c4),
      make_tc<2, 3, 14, 64, ACT_RELU, 4, true>("tc05_14x64x64x3_relu_f32lat", d_c3),
      make_tc<1, 3, 7, 48, ACT_GELU, 4, true, false, false, 40>("tc05_7x40x40x3_gelu_f32lat", d_c2),
      make_tc<1, 3, 4, 16, ACT_RELU, 4, true>("tc05_4x16x16x3_relu_f32lat", d_c1),
  };
  const int n = static_cast<int>(sizeof(list) / sizeof(list[0]));
  int k = 0;
  for (; k < n && k < cap; ++k) out[k] = list[k];
  return k;
}

}  // namespace pic
