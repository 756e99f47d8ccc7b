// k_tc_tma.cu -- the tensor-core decode kernel (k_tc.cuh) with its latents
// staged by TMA, for int32 latent symbols, one instantiation per decode
// workload architecture (its own translation unit, compiled in parallel).
#include "k_tc.cuh"

namespace pic {
namespace {
const int d_c1[] = {4, 16, 16, 3};
const int d_c2[] = {7, 40, 40, 3};
const int d_c3[] = {14, 64, 64, 3};
const int d_c4[] = {16, 64, 64, 64, 3};
const int d_c5[] = {7, 64, 64, 3};
}  // namespace

// PIC_STAGING_AUTO takes the TMA kernel where runs on GB300 measured it as
// fast as the per-thread-copy kernel (4-16-16-3: equal) and keeps the copies
// where TMA was slower (7-64-64-3: 2.7-8 %, 14-64-64-3: 1-2 %, 7-40-40-3
// GELU: 0-5 %, 16-64-64-64-3 GELU: 0-5 % from run to run).
KernelInfo tma_auto(KernelInfo k, bool on) {
  k.tma_default = on ? 1 : 0;
  return k;
}

int tc_kernels_tma(KernelInfo* out, int cap) {
  const KernelInfo list[] = {
      tma_auto(make_tc<1, 3, 7, 64, ACT_RELU, 4, false, true>("tc05_7x64x64x3_relu_tma", d_c5), false),
      tma_auto(make_tc<2, 4, 16, 64, ACT_GELU, 4, false, true>("tc05_16x64x64x64x3_gelu_tma", d_c4), false),
      tma_auto(make_tc<2, 3, 14, 64, ACT_RELU, 4, false, true>("tc05_14x64x64x3_relu_tma", d_c3), false),
      tma_auto(make_tc<1, 3, 7, 48, ACT_GELU, 4, false, true, false, 40>("tc05_7x40x40x3_gelu_tma", d_c2), false),
      tma_auto(make_tc<1, 3, 4, 16, ACT_RELU, 4, false, true>("tc05_4x16x16x3_relu_tma", d_c1), true),
  };
  const int n = static_cast<int>(sizeof(list) / sizeof(list[0]));
  int k = 0;
  for (; k < n && k < cap; ++k) out[k] = list[k];
  return k;
}

}  // namespace pic
