// pic_kernels.h -- internal registry of the decode kernels (not part of the
// public C ABI).  Each kernel translation unit lists its instantiations here;
// pic_decode.cu picks one at create time.
#pragma once

namespace pic {

struct KernelInfo {
  const char* name;
  int precision;   // 0 = fp32 CUDA cores, 1 = fp16 tensor cores
  int latent_format;  // 0 = int32 symbols, 1 = fp32 values
  int generic;     // 1: runtime dims (fallback), 0: dims fixed below
  int C;
  int n_layers;
  int dims[7];
  int act;
  int threads;     // threads per CTA
  int regs_at_launch;  // registers per thread the kernel must be built with (0: any)
  int smem_bytes;  // dynamic shared memory per CTA
  int tile_px;     // pixels per tile (one tile = a run of one image row)
  int tma;         // 1: stages the latents with TMA (needs valid TmaParams)
  int tma_default; // (TMA kernels) 1: PIC_STAGING_AUTO picks it over its per-thread-copy twin
  const void* fn;  // __global__ function taking (DecodeParams), or (DecodeParams,
                   // TmaParams) for the tensor-core kernels (precision 1)
};

int fp32_kernels(KernelInfo* out, int cap);        // all of them
int fp32_kernels_sweep(KernelInfo* out, int cap);  // the width ablation's (own translation unit)
KernelInfo fp32_generic_kernel_info(int latent_format);
int tc_kernels(KernelInfo* out, int cap);     // both latent formats
int tc_kernels_fp32lat(KernelInfo* out, int cap);  // the fp32-latent ones (own translation unit)
int tc_kernels_sweep(KernelInfo* out, int cap);    // the width ablation's (own translation unit)
int tc_kernels_tma(KernelInfo* out, int cap);      // TMA-staged variants (own translation unit)

}  // namespace pic
