// k_tc_sweep.cu -- instantiations of the tensor-core decode kernel
// (k_tc.cuh) for the width ablation's architectures: 8 single-channel
// levels and a 4-layer MLP 8-w-w-w-3 with ReLU, w = 8, 16, 32, 64.  Width 8
// runs on N = 16 tiles with the extra rows and columns zero, as the paper
// does on its tensor cores (Sec. 4.3).
#include "k_tc.cuh"

namespace pic {
namespace {
const int d_w8[] = {8, 8, 8, 8, 3};
const int d_w16[] = {8, 16, 16, 16, 3};
const int d_w32[] = {8, 32, 32, 32, 3};
const int d_w64[] = {8, 64, 64, 64, 3};
}  // namespace

int tc_kernels_sweep(KernelInfo* out, int cap) {
  const KernelInfo list[] = {
      make_tc<1, 4, 8, 16, ACT_RELU, 4, false, false, false, 8>("tc05_8x8x8x8x3_relu", d_w8),
      make_tc<1, 4, 8, 16, ACT_RELU, 4, false>("tc05_8x16x16x16x3_relu", d_w16),
      make_tc<1, 4, 8, 32, ACT_RELU, 4, false>("tc05_8x32x32x32x3_relu", d_w32),
      make_tc<1, 4, 8, 64, ACT_RELU, 4, false>("tc05_8x64x64x64x3_relu", d_w64),
  };
  const int n = static_cast<int>(sizeof(list) / sizeof(list[0]));
  int k = 0;
  for (; k < n && k < cap; ++k) out[k] = list[k];
  return k;
}

}  // namespace pic
