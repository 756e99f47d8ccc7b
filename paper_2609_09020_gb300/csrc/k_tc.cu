// k_tc.cu -- instantiations of the tensor-core decode kernel (k_tc.cuh) for
// int32 latent symbols, one per decode workload architecture, and the
// registry of both latent formats.
#include "k_tc.cuh"

namespace pic {
namespace {
const int d_c1[] = {4, 16, 16, 3};
const int d_c2[] = {7, 40, 40, 3};
const int d_c3[] = {14, 64, 64, 3};
const int d_c4[] = {16, 64, 64, 64, 3};
const int d_c5[] = {7, 64, 64, 3};
}  // namespace

int tc_kernels(KernelInfo* out, int cap) {
  const KernelInfo list[] = {
      make_tc<1, 3, 7, 64, ACT_RELU, 4, false>("tc05_7x64x64x3_relu", d_c5),
      make_tc<1, 3, 7, 64, ACT_RELU, 4, false, false, true>("tc05_7x64x64x3_relu_lo8", d_c5),
      make_tc<2, 4, 16, 64, ACT_GELU, 4, false>("tc05_16x64x64x64x3_gelu", d_c4),
      make_tc<2, 3, 14, 64, ACT_RELU, 4, false>("tc05_14x64x64x3_relu", d_c3),
      make_tc<1, 3, 7, 48, ACT_GELU, 4, false, false, false, 40>("tc05_7x40x40x3_gelu", d_c2),
      make_tc<1, 3, 4, 16, ACT_RELU, 4, false>("tc05_4x16x16x3_relu", d_c1),
  };
  const int n = static_cast<int>(sizeof(list) / sizeof(list[0]));
  int k = 0;
  for (; k < n && k < cap; ++k) out[k] = list[k];
  if (k < cap) k += tc_kernels_tma(out + k, cap - k);
  if (k < cap) k += tc_kernels_fp32lat(out + k, cap - k);
  if (k < cap) k += tc_kernels_sweep(out + k, cap - k);
  return k;
}

}  // namespace pic
