// pic_decode.cu -- the C ABI (include/pic_decode.h): argument validation,
// kernel selection, launch.  Host code only; the kernels live in k_*.cu.
#include <cstdint>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <atomic>
#include <mutex>
#include <new>

#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include "pic_common.cuh"
#include "pic_kernels.h"
#include "pic_decode.h"

using pic::DecodeParams;
using pic::KernelInfo;

struct pic_decoder {
  pic_arch arch;
  int device;
  int sm_count;
  KernelInfo kern;
  int grid_cap;          // resident CTAs over all SMs
  // the TMA-staged twin of kern (tensor-core archs that have one), launched
  // whenever the call's latent buffer can be described by tensor maps
  bool has_tma;
  KernelInfo kern_tma;
  int grid_cap_tma;
  // the last call's tensor map (it depends on the latent buffer and its size only)
  const int32_t* tma_key_ptr;
  long long tma_key_words;
  pic::TmaParams tma_cache;
  int* d_status;         // bounded-wait failure flag (device word)
  long long n_params;    // per image
  // staging for pic_decode_batch_host (allocated on first use): one region
  // per chunk of images, each starting on a 256-byte boundary
  unsigned char* s_lat;
  unsigned char* s_steps;
  unsigned char* s_w;
  unsigned char* s_out;
  // its copy-in / decode / copy-out pipeline (created on first use)
  cudaStream_t p_in, p_run, p_out;
  cudaEvent_t p_ev[3 * 16 + 1];
  bool p_ready;
};

namespace {

// Test hook of the bounded device-side waits (pic_decode_test_wait_fault):
// nonzero only while a test makes a wait run out on purpose.
std::atomic<int> g_test_fault{0};
std::atomic<unsigned> g_test_spin_limit{0};

int level_size(int n, int l) { return static_cast<int>((static_cast<long long>(n) + (1LL << l) - 1) >> l); }

bool arch_valid(const pic_arch* a) {
  if (a->num_levels < 1 || a->num_levels > pic::kMaxLevels) return false;
  if (a->channels_per_level < 1 || a->channels_per_level > 4) return false;
  if (a->num_layers < 1 || a->num_layers > pic::kMaxLayers) return false;
  if (a->dims[0] != a->num_levels * a->channels_per_level) return false;
  if (a->dims[a->num_layers] != 3) return false;
  for (int k = 0; k <= a->num_layers; ++k)
    if (a->dims[k] < 1 || a->dims[k] > pic::kMaxDim) return false;
  if (a->hidden_act != PIC_ACT_RELU && a->hidden_act != PIC_ACT_GELU) return false;
  if (a->precision != PIC_PREC_FP32 && a->precision != PIC_PREC_FP16_TC &&
      a->precision != PIC_PREC_FP16_TC_LO8)
    return false;
  if (a->clamp_output != 0 && a->clamp_output != 1) return false;
  if (a->max_H < 1 || a->max_W < 1 || a->max_batch < 1) return false;
  if (a->max_H > 65536 || a->max_W > 65536 || a->max_batch > 65536) return false;
  if (a->latent_format != PIC_LATENT_INT32 && a->latent_format != PIC_LATENT_FP32) return false;
  if (a->output_format < PIC_OUT_F32_CHW || a->output_format > PIC_OUT_U8_HWC) return false;
  if (a->staging < PIC_STAGING_AUTO || a->staging > PIC_STAGING_TMA) return false;
  return true;
}

bool kernel_matches(const KernelInfo& k, const pic_arch* a, bool tma = false) {
  if (k.generic || (k.tma != 0) != tma || k.precision != a->precision ||
      k.latent_format != a->latent_format ||
      k.C != a->channels_per_level ||
      k.n_layers != a->num_layers || k.act != a->hidden_act)
    return false;
  for (int i = 0; i <= a->num_layers; ++i)
    if (k.dims[i] != a->dims[i]) return false;
  return true;
}

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

int check_decode_args(const pic_decoder* h, int B, const int32_t* latents, const float* steps,
                      const void* weights, int H, int W, const void* out) {
  const bool need_steps = h && h->arch.latent_format == PIC_LATENT_INT32;
  if (!h || !latents || (need_steps && !steps) || !weights || !out) return PIC_ERR_INVALID_ARG;
  if (B < 1 || B > h->arch.max_batch) return PIC_ERR_INVALID_ARG;
  if (H < 1 || W < 1 || H > h->arch.max_H || W > h->arch.max_W) return PIC_ERR_INVALID_ARG;
  if (!aligned(latents, 16) || !aligned(weights, 16) || !aligned(out, 16) || !aligned(steps, 4))
    return PIC_ERR_INVALID_ARG;
  // The kernel would run on the current device with the handle's setup (and,
  // for a handle, its status word) from another: refuse instead.
  int cur = -1;
  if (cudaGetDevice(&cur) != cudaSuccess) {
    cudaGetLastError();
    return PIC_ERR_CUDA;
  }
  if (cur != h->device) return PIC_ERR_INVALID_ARG;
  return PIC_OK;
}

// cuTensorMapEncodeTiled from the driver, through the runtime (no link
// against the driver library); null if the driver does not offer it.
PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static const PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q = cudaDriverEntryPointSymbolNotFound;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess) {
      cudaGetLastError();
      f = nullptr;
    }
    return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
  }();
  return fn;
}

// Tensor map for a TMA-staged tensor-core kernel (Sec. 3.1, Eq. 1: the
// full-resolution level of image b is a C x H x W grid inside the call's
// latent buffer): the whole buffer as one 1-D tensor of 4-byte words with
// boxes of kTmaRowBox words, one box per tile row segment and channel.  Box
// coordinates are 32-bit word indices, so the buffer must hold fewer than
// 2^31 words; else (or if the driver offers no encoder, or the encode
// fails) the caller launches the per-thread-copy kernel instead.
bool encode_latent_map(pic::TmaParams& tp, const DecodeParams& p) {
  const PFN_cuTensorMapEncodeTiled_v12000 enc = tensor_map_encoder();
  const long long words = p.lat_per_image * p.B;
  if (!enc || words < 1 || words >= (1LL << 31)) return false;
  const cuuint64_t dim[1] = {static_cast<cuuint64_t>(words)};
  const cuuint64_t stride[1] = {4};  // unused for a 1-D tensor
  const cuuint32_t box[1] = {static_cast<cuuint32_t>(pic::kTmaRowBox)};
  const cuuint32_t elem_stride[1] = {1u};
  return enc(&tp.lat, CU_TENSOR_MAP_DATA_TYPE_INT32, 1, const_cast<int32_t*>(p.latents), dim, stride,
             box, elem_stride, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
             CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

void fill_params(const pic_decoder* h, DecodeParams& p, int B, const int32_t* latents,
                 const float* steps, const void* weights, int H, int W, void* out) {
  std::memset(&p, 0, sizeof(p));
  const pic_arch& a = h->arch;
  p.latents = latents;
  p.steps = steps;
  p.weights = weights;
  p.out = out;
  p.H = H;
  p.W = W;
  p.B = B;
  p.L = a.num_levels;
  p.C = a.channels_per_level;
  p.clamp = a.clamp_output;
  p.out_format = a.output_format;
  p.status = h->d_status;
  p.n_layers = a.num_layers;
  for (int k = 0; k <= a.num_layers; ++k) p.dims[k] = a.dims[k];
  p.act = a.hidden_act;
  long long off = 0;
  for (int l = 0; l < a.num_levels; ++l) {
    pic::LevelGeom& g = p.lv[l];
    g.H = level_size(H, l);
    g.W = level_size(W, l);
    g.off = off;
    g.sx = static_cast<float>(static_cast<double>(g.W) / W);
    g.sy = static_cast<float>(static_cast<double>(g.H) / H);
    off += static_cast<long long>(a.channels_per_level) * g.H * g.W;
  }
  p.lat_per_image = off;
  p.params_per_image = h->n_params;
  const int tp = h->kern.tile_px;
  p.tiles_per_row = (W + tp - 1) / tp;
  p.tiles_per_image = static_cast<long long>(p.tiles_per_row) * H;
  p.total_tiles = p.tiles_per_image * B;
  const unsigned test_limit = g_test_spin_limit.load(std::memory_order_relaxed);
  p.spin_limit = test_limit ? test_limit : pic::kWaitPolls;
  p.test_fault = g_test_fault.load(std::memory_order_relaxed);
}

int launch(pic_decoder* h, const DecodeParams& p, cudaStream_t stream) {
  const KernelInfo* k = &h->kern;
  int cap = h->grid_cap;
  // tensor-core kernels take the tensor maps as a second parameter (unused
  // by the per-thread-copy kernels, but always passed, zeroed)
  static const pic::TmaParams kNoMaps{};
  const pic::TmaParams* tp = &kNoMaps;
  if (h->has_tma) {
    const long long words = p.lat_per_image * p.B;
    bool ok = h->tma_key_ptr == p.latents && h->tma_key_words == words;
    if (!ok) {
      h->tma_key_ptr = nullptr;
      ok = encode_latent_map(h->tma_cache, p);
      if (ok) {
        h->tma_key_ptr = p.latents;
        h->tma_key_words = words;
      }
    }
    if (ok) {
      k = &h->kern_tma;
      cap = h->grid_cap_tma;
      tp = &h->tma_cache;
    }
  }
  long long grid = p.total_tiles < cap ? p.total_tiles : cap;
  if (grid < 1) grid = 1;
  void* args[] = {const_cast<DecodeParams*>(&p), const_cast<pic::TmaParams*>(tp)};
  cudaError_t e = cudaLaunchKernel(k->fn, dim3(static_cast<unsigned>(grid)), dim3(k->threads), args,
                                   k->smem_bytes, stream);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return PIC_ERR_CUDA;
  }
  return PIC_OK;
}

size_t weight_elem_bytes(const pic_arch& a) { return a.precision == PIC_PREC_FP32 ? 4 : 2; }

// A kernel that moves registers between its warpgroups at run time assumes
// the register count it was launched with; any other build is refused
// (its register increase could otherwise never be granted).
bool regs_match(const pic::KernelInfo& k) {
  if (k.regs_at_launch == 0) return true;
  cudaFuncAttributes a{};
  if (cudaFuncGetAttributes(&a, k.fn) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.numRegs == k.regs_at_launch;
}

}  // namespace

extern "C" {

const char* pic_status_string(int s) {
  switch (s) {
    case PIC_OK: return "ok";
    case PIC_ERR_INVALID_ARG: return "invalid argument";
    case PIC_ERR_UNSUPPORTED: return "unsupported architecture or device";
    case PIC_ERR_CUDA: return "CUDA error";
    case PIC_ERR_ALLOC: return "allocation failed";
    case PIC_ERR_TIMEOUT: return "device-side wait timed out";
    default: return "unknown status";
  }
}

int64_t pic_latent_count(int H, int W, int L, int C) {
  if (H < 1 || W < 1 || L < 1 || L > 30 || C < 1) return -1;
  int64_t n = 0;
  for (int l = 0; l < L; ++l) n += static_cast<int64_t>(C) * level_size(H, l) * level_size(W, l);
  return n;
}

int64_t pic_param_count(const pic_arch* a) {
  if (!a || a->num_layers < 1 || a->num_layers > pic::kMaxLayers) return -1;
  int64_t n = 0;
  for (int k = 0; k < a->num_layers; ++k) {
    if (a->dims[k] < 1 || a->dims[k + 1] < 1) return -1;
    n += static_cast<int64_t>(a->dims[k + 1]) * (a->dims[k] + 1);
  }
  return n;
}

int pic_decode_create(const pic_arch* arch, pic_decoder** out) {
  if (!out) return PIC_ERR_INVALID_ARG;
  *out = nullptr;
  if (!arch) return PIC_ERR_INVALID_ARG;
  if (arch->num_layers < 1 || arch->num_layers > pic::kMaxLayers) return PIC_ERR_INVALID_ARG;
  if (arch->dims[0] != arch->num_levels * arch->channels_per_level ||
      arch->dims[arch->num_layers] != 3)
    return PIC_ERR_INVALID_ARG;
  if (!arch_valid(arch)) return PIC_ERR_UNSUPPORTED;

  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return PIC_ERR_UNSUPPORTED;
  }
  cudaDeviceProp prop;
  if (cudaGetDeviceProperties(&prop, dev) != cudaSuccess) {
    cudaGetLastError();
    return PIC_ERR_CUDA;
  }
  if (prop.major != 10 || prop.minor != 3) return PIC_ERR_UNSUPPORTED;  // built for sm_103a only

  // Kernel selection: a compile-time specialisation of exactly this arch,
  // else (fp32 only) the generic kernel.
  KernelInfo table[32];
  int n = arch->precision == PIC_PREC_FP32 ? pic::fp32_kernels(table, 32) : pic::tc_kernels(table, 32);
  const KernelInfo* chosen = nullptr;
  for (int i = 0; i < n && i < 32; ++i)
    if (kernel_matches(table[i], arch)) {
      chosen = &table[i];
      break;
    }
  KernelInfo k{};
  if (chosen) {
    k = *chosen;
  } else if (arch->precision == PIC_PREC_FP32) {
    k = pic::fp32_generic_kernel_info(arch->latent_format);
    k.smem_bytes = static_cast<int>(pic_param_count(arch) * 4);
  } else {
    return PIC_ERR_UNSUPPORTED;
  }
  if (k.smem_bytes > static_cast<int>(prop.sharedMemPerBlockOptin)) return PIC_ERR_UNSUPPORTED;
  if (!regs_match(k)) return PIC_ERR_UNSUPPORTED;
  if (cudaFuncSetAttribute(k.fn, cudaFuncAttributeMaxDynamicSharedMemorySize, k.smem_bytes) !=
      cudaSuccess) {
    cudaGetLastError();
    return PIC_ERR_CUDA;
  }
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k.fn, k.threads, k.smem_bytes) !=
          cudaSuccess ||
      per_sm < 1) {
    cudaGetLastError();
    return PIC_ERR_UNSUPPORTED;
  }

  // the TMA-staged twin, where the arch has one
  const KernelInfo* twin = nullptr;
  int per_sm_tma = 0;
  for (int i = 0; i < n && i < 32; ++i)
    if (kernel_matches(table[i], arch, true)) {
      twin = &table[i];
      break;
    }
  if (arch->staging == PIC_STAGING_COPIES || (arch->staging == PIC_STAGING_AUTO && twin && !twin->tma_default))
    twin = nullptr;
  if (arch->staging == PIC_STAGING_TMA && !twin) return PIC_ERR_UNSUPPORTED;
  if (twin && (twin->smem_bytes > static_cast<int>(prop.sharedMemPerBlockOptin) || !regs_match(*twin) ||
               cudaFuncSetAttribute(twin->fn, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    twin->smem_bytes) != cudaSuccess ||
               cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm_tma, twin->fn, twin->threads,
                                                             twin->smem_bytes) != cudaSuccess ||
               per_sm_tma < 1)) {
    cudaGetLastError();
    if (arch->staging == PIC_STAGING_TMA) return PIC_ERR_UNSUPPORTED;
    twin = nullptr;  // the per-thread-copy kernel serves every call
  }

  pic_decoder* h = new (std::nothrow) pic_decoder();
  if (!h) return PIC_ERR_ALLOC;
  h->arch = *arch;
  h->device = dev;
  h->sm_count = prop.multiProcessorCount;
  h->kern = k;
  h->grid_cap = per_sm * prop.multiProcessorCount;
  if (twin) {
    h->has_tma = true;
    h->kern_tma = *twin;
    h->grid_cap_tma = per_sm_tma * prop.multiProcessorCount;
  }
  h->n_params = pic_param_count(arch);
  if (cudaMalloc(&h->d_status, sizeof(int)) != cudaSuccess) {
    cudaGetLastError();
    delete h;
    return PIC_ERR_ALLOC;
  }
  if (cudaMemset(h->d_status, 0, sizeof(int)) != cudaSuccess) {
    cudaGetLastError();
    cudaFree(h->d_status);
    delete h;
    return PIC_ERR_CUDA;
  }
  *out = h;
  return PIC_OK;
}

int pic_decode_batch(pic_decoder* h, int B, const int32_t* latents, const float* steps,
                     const void* weights, int H, int W, void* out_rgb, void* stream) {
  int rc = check_decode_args(h, B, latents, steps, weights, H, W, out_rgb);
  if (rc != PIC_OK) return rc;
  DecodeParams p;
  fill_params(h, p, B, latents, steps, weights, H, W, out_rgb);
  return launch(h, p, static_cast<cudaStream_t>(stream));
}

int pic_decode(pic_decoder* h, const int32_t* latents, const float* steps, const void* weights,
               int H, int W, void* out_rgb, void* stream) {
  return pic_decode_batch(h, 1, latents, steps, weights, H, W, out_rgb, stream);
}

}  // extern "C"

namespace {

constexpr int kHostChunks = 16;  // pipeline depth of pic_decode_batch_host
constexpr long long kChunkAlign = 256;

long long align_up(long long v, long long a) { return (v + a - 1) / a * a; }

// Bytes of a staging buffer holding `per_image` bytes for each of `imgs`
// images in up to kHostChunks chunks, each chunk starting on a
// kChunkAlign-byte boundary.
long long staging_bytes(long long per_image, int imgs) {
  return align_up(per_image * imgs, kChunkAlign) + kHostChunks * kChunkAlign;
}

// Chunks of pic_decode_batch_host: image b0[c] .. b0[c+1] - 1 for chunk c.
// The first chunks are one and two images, so that the copy-back (the
// slowest stage: fp32 RGB is the largest buffer) starts after one image has
// been copied in and decoded; the rest of the batch is split evenly over the
// remaining chunks.  Returns the number of chunks.
int host_chunks(int B, int (&b0)[kHostChunks + 1]) {
  int n = 0, b = 0;
  b0[0] = 0;
  for (const int first : {1, 2}) {
    if (b >= B) break;
    b += first < B - b ? first : B - b;
    b0[++n] = b;
  }
  const int left = B - b, rest = kHostChunks - n;
  for (int i = 1; i <= rest && b < B; ++i) {
    const int e = (B - left) + static_cast<int>(static_cast<long long>(left) * i / rest);
    if (e > b) b0[++n] = b = e;
  }
  return n;
}

void free_host_pipeline(pic_decoder* h) {
  cudaFree(h->s_lat);
  cudaFree(h->s_steps);
  cudaFree(h->s_w);
  cudaFree(h->s_out);
  h->s_lat = h->s_steps = h->s_w = h->s_out = nullptr;
  if (h->p_ready) {
    cudaStreamDestroy(h->p_in);
    cudaStreamDestroy(h->p_run);
    cudaStreamDestroy(h->p_out);
    for (cudaEvent_t& e : h->p_ev) cudaEventDestroy(e);
    h->p_ready = false;
  }
  cudaGetLastError();
}

}  // namespace

extern "C" {

/*
 * Host-buffer decode as a three-stage pipeline over chunks of images: the
 * inputs of chunk c go to the device on one stream while chunk c - 1 decodes
 * on a second and chunk c - 2's RGB returns on a third, so the host<->device
 * copies overlap each other and the kernels instead of adding up.
 */
int pic_decode_batch_host(pic_decoder* h, int B, const int32_t* latents, const float* steps,
                          const void* weights, int H, int W, void* out_rgb, void* stream) {
  if (!h || !latents || (h->arch.latent_format == PIC_LATENT_INT32 && !steps) || !weights ||
      !out_rgb)
    return PIC_ERR_INVALID_ARG;
  if (B < 1 || B > h->arch.max_batch || H < 1 || W < 1 || H > h->arch.max_H || W > h->arch.max_W)
    return PIC_ERR_INVALID_ARG;
  const pic_arch& a = h->arch;
  const long long out_elem = a.output_format == PIC_OUT_U8_HWC ? 1 : 4;
  if (!h->s_lat) {
    const long long lat = pic_latent_count(a.max_H, a.max_W, a.num_levels, a.channels_per_level);
    bool ok =
        cudaMalloc(&h->s_lat, staging_bytes(lat * 4, a.max_batch)) == cudaSuccess &&
        cudaMalloc(&h->s_steps, staging_bytes(a.num_levels * 4LL, a.max_batch)) == cudaSuccess &&
        cudaMalloc(&h->s_w, staging_bytes(h->n_params * static_cast<long long>(weight_elem_bytes(a)),
                                          a.max_batch)) == cudaSuccess &&
        cudaMalloc(&h->s_out, staging_bytes(3LL * a.max_H * a.max_W * 4, a.max_batch)) == cudaSuccess;
    if (ok && !h->p_ready) {
      ok = cudaStreamCreateWithFlags(&h->p_in, cudaStreamNonBlocking) == cudaSuccess &&
           cudaStreamCreateWithFlags(&h->p_run, cudaStreamNonBlocking) == cudaSuccess &&
           cudaStreamCreateWithFlags(&h->p_out, cudaStreamNonBlocking) == cudaSuccess;
      for (cudaEvent_t& e : h->p_ev)
        ok = ok && cudaEventCreateWithFlags(&e, cudaEventDisableTiming) == cudaSuccess;
      h->p_ready = ok;
    }
    if (!ok) {
      free_host_pipeline(h);
      return PIC_ERR_ALLOC;
    }
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const long long lat_img = pic_latent_count(H, W, a.num_levels, a.channels_per_level) * 4;
  const long long st_img = a.num_levels * 4LL;
  const long long w_img = h->n_params * static_cast<long long>(weight_elem_bytes(a));
  const long long out_img = 3LL * H * W * out_elem;
  int b0s[kHostChunks + 1];
  const int n_chunks = host_chunks(B, b0s);
  const bool have_steps = steps != nullptr;
  cudaEvent_t* ev = h->p_ev;  // [0]: start; then (in, run, out) per chunk

  auto cuda_fail = [&]() {
    cudaGetLastError();
    return PIC_ERR_CUDA;
  };
  if (cudaEventRecord(ev[0], s) != cudaSuccess || cudaStreamWaitEvent(h->p_in, ev[0], 0) != cudaSuccess)
    return cuda_fail();
  // chunk c's staging starts on a kChunkAlign boundary after chunk c - 1's
  long long o_lat = 0, o_st = 0, o_w = 0, o_out = 0;
  int c = 0;
  for (; c < n_chunks; ++c) {
    const int b0 = b0s[c], nb = b0s[c + 1] - b0s[c];
    unsigned char* d_lat = h->s_lat + o_lat;
    unsigned char* d_st = h->s_steps + o_st;
    unsigned char* d_w = h->s_w + o_w;
    unsigned char* d_out = h->s_out + o_out;
    o_lat = align_up(o_lat + nb * lat_img, kChunkAlign);
    o_st = align_up(o_st + nb * st_img, kChunkAlign);
    o_w = align_up(o_w + nb * w_img, kChunkAlign);
    o_out = align_up(o_out + nb * out_img, kChunkAlign);
    cudaEvent_t e_in = ev[1 + 3 * c], e_run = ev[2 + 3 * c], e_out = ev[3 + 3 * c];
    if (cudaMemcpyAsync(d_lat, reinterpret_cast<const unsigned char*>(latents) + b0 * lat_img, nb * lat_img,
                        cudaMemcpyHostToDevice, h->p_in) != cudaSuccess ||
        (have_steps && cudaMemcpyAsync(d_st, reinterpret_cast<const unsigned char*>(steps) + b0 * st_img,
                                       nb * st_img, cudaMemcpyHostToDevice, h->p_in) != cudaSuccess) ||
        cudaMemcpyAsync(d_w, static_cast<const unsigned char*>(weights) + b0 * w_img, nb * w_img,
                        cudaMemcpyHostToDevice, h->p_in) != cudaSuccess ||
        cudaEventRecord(e_in, h->p_in) != cudaSuccess ||
        cudaStreamWaitEvent(h->p_run, e_in, 0) != cudaSuccess)
      return cuda_fail();
    const int rc = pic_decode_batch(h, nb, reinterpret_cast<const int32_t*>(d_lat),
                                    have_steps ? reinterpret_cast<const float*>(d_st) : nullptr, d_w, H,
                                    W, d_out, h->p_run);
    if (rc != PIC_OK) return rc;
    if (cudaEventRecord(e_run, h->p_run) != cudaSuccess ||
        cudaStreamWaitEvent(h->p_out, e_run, 0) != cudaSuccess ||
        cudaMemcpyAsync(static_cast<unsigned char*>(out_rgb) + b0 * out_img, d_out, nb * out_img,
                        cudaMemcpyDeviceToHost, h->p_out) != cudaSuccess ||
        cudaEventRecord(e_out, h->p_out) != cudaSuccess)
      return cuda_fail();
  }
  // every copy-out is on p_out in order: the caller's stream waits for the last
  if (cudaStreamWaitEvent(s, ev[3 * c], 0) != cudaSuccess || cudaStreamSynchronize(s) != cudaSuccess)
    return cuda_fail();
  return PIC_OK;
}

int pic_decode_check(pic_decoder* h, void* stream) {
  if (!h) return PIC_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int flag = 0;
  if (cudaMemcpyAsync(&flag, h->d_status, sizeof(int), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess) {
    cudaGetLastError();
    return PIC_ERR_CUDA;
  }
  if (flag != 0) {
    if (cudaMemsetAsync(h->d_status, 0, sizeof(int), s) != cudaSuccess ||
        cudaStreamSynchronize(s) != cudaSuccess) {
      cudaGetLastError();
      return PIC_ERR_CUDA;
    }
    return PIC_ERR_TIMEOUT;
  }
  return PIC_OK;
}

int pic_decode_test_wait_fault(int withhold_arrival, unsigned spin_limit) {
  if (withhold_arrival != 0 && withhold_arrival != 1) return PIC_ERR_INVALID_ARG;
  g_test_spin_limit.store(spin_limit, std::memory_order_relaxed);
  g_test_fault.store(withhold_arrival, std::memory_order_relaxed);
  return PIC_OK;
}

void pic_decode_destroy(pic_decoder* h) {
  if (!h) return;
  cudaDeviceSynchronize();
  cudaFree(h->d_status);
  free_host_pipeline(h);
  delete h;
}

const char* pic_decode_kernel_name(const pic_decoder* h) {
  if (!h) return "";
  return h->has_tma ? h->kern_tma.name : h->kern.name;
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Allocation-free entry point.
//
// Some callers cannot call cudaMalloc: a plug-in inside a host application
// that hands out all device memory from its own pool and forbids any other
// allocation, a real-time loop that cannot accept cudaMalloc's implicit
// device synchronisation and unbounded latency, or a service whose memory
// budget is fixed before it starts.  pic_decode_create() allocates (the
// handle's status word), so those callers use pic_decode_batch_noalloc()
// instead.  It runs the same kernels; the only global memory it needs beyond
// the caller's inputs and outputs -- the status word that a bounded wait in
// the tensor-core kernel raises when it gives up -- lives in the static
// device array below, which every GPU that loads this library holds until
// the process exits.  A device global is zero when the module loads, so the
// word starts at zero; pic_decode_noalloc_check() reads and clears it.
namespace {

constexpr int kStaticScratchInts = 64;  // 256 bytes; one call needs 1 word
constexpr int kMaxStaticDevices = 64;
constexpr int kNoallocKernelCache = 32;  // (device, kernel) pairs remembered

// What one device needs looked up once: its capabilities and the device
// address of the static scratch (the array's name is only a host-side
// stand-in).  Only successful look-ups are kept, so a failed first try
// (no context yet, say) is retried by the next call.
struct NoallocDevice {
  bool ready;
  int major, minor, sms, smem_optin;
  int* scratch;
};
// Per (device, kernel): the shared-memory attribute is set and the
// occupancy and register count were read.
struct NoallocKernel {
  int dev;
  const void* fn;
  int per_sm;
  bool regs_ok;
};

std::mutex g_noalloc_mutex;
NoallocDevice g_noalloc_dev[kMaxStaticDevices];
NoallocKernel g_noalloc_kern[kNoallocKernelCache];
int g_noalloc_nkern = 0;

}  // namespace

static __device__ __align__(256) int g_static_scratch[kStaticScratchInts];

namespace {

// Device facts and the static scratch address of `dev` (current), cached.
int noalloc_device(int dev, NoallocDevice* out) {
  if (dev < 0 || dev >= kMaxStaticDevices) return PIC_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_noalloc_mutex);
  NoallocDevice& d = g_noalloc_dev[dev];
  if (!d.ready) {
    NoallocDevice t{};
    void* p = nullptr;
    if (cudaDeviceGetAttribute(&t.major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&t.minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&t.sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&t.smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) !=
            cudaSuccess ||
        cudaGetSymbolAddress(&p, g_static_scratch) != cudaSuccess || p == nullptr) {
      cudaGetLastError();
      return PIC_ERR_CUDA;
    }
    t.scratch = static_cast<int*>(p);
    t.ready = true;
    d = t;
  }
  *out = d;
  return PIC_OK;
}

// Occupancy of kernel `k` on `dev` (current), after setting its shared-memory
// attribute; both done once per (device, kernel).
int noalloc_kernel(int dev, const KernelInfo& k, int* per_sm) {
  std::lock_guard<std::mutex> lock(g_noalloc_mutex);
  for (int i = 0; i < g_noalloc_nkern; ++i)
    if (g_noalloc_kern[i].dev == dev && g_noalloc_kern[i].fn == k.fn) {
      if (!g_noalloc_kern[i].regs_ok) return PIC_ERR_UNSUPPORTED;
      *per_sm = g_noalloc_kern[i].per_sm;
      return PIC_OK;
    }
  NoallocKernel e{dev, k.fn, 0, regs_match(k)};
  if (e.regs_ok) {
    if (cudaFuncSetAttribute(k.fn, cudaFuncAttributeMaxDynamicSharedMemorySize, k.smem_bytes) !=
        cudaSuccess) {
      cudaGetLastError();
      return PIC_ERR_CUDA;
    }
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&e.per_sm, k.fn, k.threads, k.smem_bytes) !=
            cudaSuccess ||
        e.per_sm < 1) {
      cudaGetLastError();
      return PIC_ERR_UNSUPPORTED;
    }
  }
  if (g_noalloc_nkern < kNoallocKernelCache) g_noalloc_kern[g_noalloc_nkern++] = e;
  if (!e.regs_ok) return PIC_ERR_UNSUPPORTED;
  *per_sm = e.per_sm;
  return PIC_OK;
}

}  // namespace

extern "C" int pic_decode_batch_noalloc(const pic_arch* arch, int B, const int32_t* latents,
                                        const float* steps, const void* weights, int H, int W,
                                        void* out_rgb, void* stream) {
  if (!arch) return PIC_ERR_INVALID_ARG;
  if (arch->num_layers < 1 || arch->num_layers > pic::kMaxLayers) return PIC_ERR_INVALID_ARG;
  if (arch->dims[0] != arch->num_levels * arch->channels_per_level ||
      arch->dims[arch->num_layers] != 3)
    return PIC_ERR_INVALID_ARG;
  if (!arch_valid(arch)) return PIC_ERR_UNSUPPORTED;
  // Scratch needed by one call: the status word.  Anything that would need
  // more than the static array holds is refused.
  constexpr int kNeededInts = 1;
  static_assert(kNeededInts <= kStaticScratchInts, "static scratch too small");

  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return PIC_ERR_UNSUPPORTED;
  }
  NoallocDevice d{};
  int rc = noalloc_device(dev, &d);
  if (rc != PIC_OK) return rc;
  if (d.major != 10 || d.minor != 3) return PIC_ERR_UNSUPPORTED;

  // The same kernel selection as pic_decode_create, on a handle that lives
  // on this stack frame.
  KernelInfo table[32];
  int n = arch->precision == PIC_PREC_FP32 ? pic::fp32_kernels(table, 32) : pic::tc_kernels(table, 32);
  const KernelInfo* chosen = nullptr;
  for (int i = 0; i < n && i < 32; ++i)
    if (kernel_matches(table[i], arch)) {
      chosen = &table[i];
      break;
    }
  pic_decoder h{};
  h.arch = *arch;
  h.device = dev;
  h.sm_count = d.sms;
  if (chosen) {
    h.kern = *chosen;
  } else if (arch->precision == PIC_PREC_FP32) {
    h.kern = pic::fp32_generic_kernel_info(arch->latent_format);
    h.kern.smem_bytes = static_cast<int>(pic_param_count(arch) * 4);
  } else {
    return PIC_ERR_UNSUPPORTED;
  }
  if (h.kern.smem_bytes > d.smem_optin) return PIC_ERR_UNSUPPORTED;
  rc = check_decode_args(&h, B, latents, steps, weights, H, W, out_rgb);
  if (rc != PIC_OK) return rc;
  int per_sm = 0;
  rc = noalloc_kernel(dev, h.kern, &per_sm);
  if (rc != PIC_OK) return rc;
  h.grid_cap = per_sm * d.sms;
  // the TMA-staged twin, as pic_decode_create picks it (its tensor maps are
  // encoded on the host for each call: no device memory)
  for (int i = 0; i < n && i < 32; ++i)
    if (kernel_matches(table[i], arch, true)) {
      if (arch->staging == PIC_STAGING_COPIES ||
          (arch->staging == PIC_STAGING_AUTO && !table[i].tma_default))
        break;
      int per_sm_tma = 0;
      if (table[i].smem_bytes <= d.smem_optin && noalloc_kernel(dev, table[i], &per_sm_tma) == PIC_OK) {
        h.has_tma = true;
        h.kern_tma = table[i];
        h.grid_cap_tma = per_sm_tma * d.sms;
      }
      break;
    }
  if (arch->staging == PIC_STAGING_TMA && !h.has_tma) return PIC_ERR_UNSUPPORTED;
  h.n_params = pic_param_count(arch);
  h.d_status = d.scratch;

  DecodeParams p;
  fill_params(&h, p, B, latents, steps, weights, H, W, out_rgb);
  return launch(&h, p, static_cast<cudaStream_t>(stream));
}

extern "C" int pic_decode_noalloc_check(void* stream) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return PIC_ERR_CUDA;
  }
  NoallocDevice d{};
  int rc = noalloc_device(dev, &d);
  if (rc != PIC_OK) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int flag = 0;
  if (cudaMemcpyAsync(&flag, d.scratch, sizeof(int), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess) {
    cudaGetLastError();
    return PIC_ERR_CUDA;
  }
  if (flag == 0) return PIC_OK;
  if (cudaMemsetAsync(d.scratch, 0, sizeof(int), s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess) {
    cudaGetLastError();
    return PIC_ERR_CUDA;
  }
  return PIC_ERR_TIMEOUT;
}
