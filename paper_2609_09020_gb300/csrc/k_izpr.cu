// k_izpr.cu -- inverse ZpR on the GPU (Sec. 3.3, Fig. 2; App. B, Algorithm 1),
// behind the C ABI of include/pic_izpr.h.
//
// 1. Marker offsets by stream compaction (the role of Algorithm 1's
//    precomputed offsets): count the eob markers of each 4096-symbol chunk,
//    exclusive-scan the chunk counts in one CTA, then write every marker's
//    stream index in stream order.
// 2. Expansion: one warp per block (Algorithm 1 uses one thread per block).
//    The lanes load the block's symbols (at most 64), each knows how many
//    positions it covers (1 for a literal, n for the run code of n zeros), a
//    warp scan turns those counts into zigzag positions, literals are
//    scattered into a zeroed 64-entry block in shared memory through the
//    zigzag table, and the block leaves as two coalesced 128-byte rows.
#include <cstdint>

#include <cuda_runtime.h>

#include "pic_decode.h"
#include "pic_izpr.h"

namespace pic {
namespace {

constexpr int kThreads = 256;
constexpr int kPerThread = 16;
constexpr int kChunk = kThreads * kPerThread;  // symbols per compaction chunk

enum : int { kBadBlock = 1, kBadCount = 2 };

// Workspace: status word, marker total, chunk counts, chunk bases.
struct Workspace {
  int* status;
  long long* total;
  int* counts;
  long long* base;
};
__host__ __device__ inline long long n_chunks_of(long long n) { return (n + kChunk - 1) / kChunk; }
__host__ __device__ inline long long ws_bytes(long long n) {
  const long long c = n_chunks_of(n);
  return 32 + ((c * 4 + 15) / 16) * 16 + c * 8;
}
__host__ __device__ inline Workspace ws_view(void* w, long long n) {
  char* p = static_cast<char*>(w);
  const long long c = n_chunks_of(n);
  Workspace v;
  v.status = reinterpret_cast<int*>(p);
  v.total = reinterpret_cast<long long*>(p + 16);
  v.counts = reinterpret_cast<int*>(p + 32);
  v.base = reinterpret_cast<long long*>(p + 32 + ((c * 4 + 15) / 16) * 16);
  return v;
}

// Zigzag order of an 8x8 block (raster index of the k-th zigzag position):
// anti-diagonal d = row + col, row falling for even d, rising for odd d.
struct ZigzagTable {
  int v[64];
};
constexpr ZigzagTable make_zigzag() {
  ZigzagTable t{};
  int k = 0;
  for (int d = 0; d < 15; ++d) {
    const int first = d < 8 ? 0 : d - 7;
    const int last = d < 8 ? d : 7;
    for (int s = 0; s <= last - first; ++s) {
      const int row = (d & 1) ? first + s : last - s;
      t.v[k++] = row * 8 + (d - row);
    }
  }
  return t;
}
__constant__ ZigzagTable kZigzag = make_zigzag();

// Exclusive scan of one int per thread over a 256-thread CTA; returns the
// thread's prefix and writes the CTA total to *total.
__device__ int cta_exclusive_scan(int v, int* smem, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) smem[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int w = lane < kThreads / 32 ? smem[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    if (lane < kThreads / 32) smem[32 + lane] = w;  // inclusive warp totals
  }
  __syncthreads();
  const int before = warp > 0 ? smem[32 + warp - 1] : 0;
  *total = smem[32 + kThreads / 32 - 1];
  __syncthreads();
  return before + x - v;
}

__global__ void __launch_bounds__(kThreads) izpr_count(const int32_t* __restrict__ sym,
                                                       long long n, int32_t eob, int* counts) {
  __shared__ int smem[64];
  const long long base = static_cast<long long>(blockIdx.x) * kChunk;
  int c = 0;
#pragma unroll
  for (int k = 0; k < kPerThread; ++k) {  // coalesced: thread t reads base + t + 256 k
    const long long i = base + threadIdx.x + static_cast<long long>(kThreads) * k;
    if (i < n && __ldg(sym + i) == eob) ++c;
  }
  int total;
  cta_exclusive_scan(c, smem, &total);
  if (threadIdx.x == 0) counts[blockIdx.x] = total;
}

// One CTA: exclusive scan of the chunk counts into chunk bases; the total.
__global__ void __launch_bounds__(1024) izpr_scan(const int* counts, long long n_chunks,
                                                  long long* base, long long* total) {
  __shared__ long long part[1024];
  const long long per = (n_chunks + 1023) / 1024;
  const long long lo = threadIdx.x * per, hi = lo + per < n_chunks ? lo + per : n_chunks;
  long long s = 0;
  for (long long j = lo; j < hi; ++j) s += counts[j];
  part[threadIdx.x] = s;
  __syncthreads();
  for (int o = 1; o < 1024; o <<= 1) {  // Hillis-Steele inclusive scan of the parts
    const long long y = threadIdx.x >= o ? part[threadIdx.x - o] : 0;
    __syncthreads();
    part[threadIdx.x] += y;
    __syncthreads();
  }
  long long run = part[threadIdx.x] - s;
  for (long long j = lo; j < hi; ++j) {
    base[j] = run;
    run += counts[j];
  }
  if (threadIdx.x == 1023) *total = part[1023];
}

__global__ void __launch_bounds__(kThreads) izpr_compact(const int32_t* __restrict__ sym,
                                                         long long n, int32_t eob,
                                                         const long long* __restrict__ base,
                                                         int64_t* offsets, long long n_blocks,
                                                         int* status) {
  __shared__ int smem[64];
  // thread t owns symbols base + 16 t .. 16 t + 15 of the chunk (stream order)
  const long long first = static_cast<long long>(blockIdx.x) * kChunk +
                          static_cast<long long>(threadIdx.x) * kPerThread;
  int c = 0;
#pragma unroll
  for (int k = 0; k < kPerThread; ++k)
    if (first + k < n && __ldg(sym + first + k) == eob) ++c;
  int total;
  int pos = cta_exclusive_scan(c, smem, &total);
  const long long b0 = base[blockIdx.x];
  for (int k = 0; k < kPerThread && c > 0; ++k) {
    const long long i = first + k;
    if (i < n && __ldg(sym + i) == eob) {
      const long long slot = b0 + pos++;
      if (slot < n_blocks) offsets[slot] = i;
      else atomicOr(status, kBadCount);
      --c;
    }
  }
}

// One warp per block (grid-stride).
__global__ void __launch_bounds__(kThreads) izpr_expand(const int32_t* __restrict__ sym,
                                                        int32_t eob,
                                                        const int64_t* __restrict__ offsets,
                                                        long long n_blocks, const long long* total,
                                                        int32_t* coeffs, int* status) {
  __shared__ int blk_s[kThreads / 32][64];
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  int* blk = blk_s[wib];
  const long long found = *total;
  if (blockIdx.x == 0 && threadIdx.x == 0 && found != n_blocks) atomicOr(status, kBadCount);
  const long long valid = found < n_blocks ? found : n_blocks;
  const long long warps = static_cast<long long>(gridDim.x) * (kThreads / 32);
  for (long long b = static_cast<long long>(blockIdx.x) * (kThreads / 32) + wib; b < n_blocks;
       b += warps) {
    blk[lane] = 0;
    blk[lane + 32] = 0;
    __syncwarp();
    if (b < valid) {
      const long long start = b == 0 ? 0 : offsets[b - 1] + 1;
      const long long len = offsets[b] - start;  // symbols before this block's marker
      bool bad = len < 0 || len > 64;
      int carry = 0;
      for (int half = 0; half < 2 && !bad; ++half) {
        const int i = lane + 32 * half;
        int s = 0, cnt = 0;
        if (i < len) {
          s = __ldg(sym + start + i);
          cnt = (s >= eob - 16 && s < eob) ? s - (eob - 17) : 1;  // run of n zeros, or a literal
          if (s >= eob) bad = true;
        }
        int x = cnt;  // inclusive scan of the covered positions
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int y = __shfl_up_sync(0xffffffffu, x, o);
          if (lane >= o) x += y;
        }
        const int pos = carry + x - cnt;
        if (pos + cnt > 64) bad = true;
        else if (cnt == 1 && i < len && !(s >= eob - 16 && s < eob)) blk[kZigzag.v[pos]] = s;
        carry += __shfl_sync(0xffffffffu, x, 31);
        bad = __any_sync(0xffffffffu, bad);
      }
      if (bad && lane == 0) atomicOr(status, kBadBlock);
    }
    __syncwarp();
    int32_t* out = coeffs + b * 64;
    out[lane] = blk[lane];
    out[lane + 32] = blk[lane + 32];
    __syncwarp();
  }
}

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

}  // namespace
}  // namespace pic

extern "C" {

int64_t pic_izpr_workspace_bytes(int64_t n_symbols) {
  if (n_symbols < 0) return -1;
  return pic::ws_bytes(n_symbols);
}

int pic_izpr_decode(const int32_t* symbols, int64_t n_symbols, int32_t eob, int64_t n_blocks,
                    int32_t* coeffs, int64_t* offsets, void* workspace, size_t workspace_bytes,
                    void* stream) {
  using namespace pic;
  if (n_symbols < 0 || n_blocks < 0) return PIC_ERR_INVALID_ARG;
  if (!workspace || !aligned(workspace, 16)) return PIC_ERR_INVALID_ARG;
  if (static_cast<long long>(workspace_bytes) < ws_bytes(n_symbols)) return PIC_ERR_INVALID_ARG;
  if ((n_symbols > 0 && (!symbols || !aligned(symbols, 4))) ||
      (n_blocks > 0 && (!coeffs || !offsets || !aligned(coeffs, 16) || !aligned(offsets, 8))))
    return PIC_ERR_INVALID_ARG;
  if (eob < INT32_MIN + 17) return PIC_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  Workspace ws = ws_view(workspace, n_symbols);
  const long long chunks = n_chunks_of(n_symbols);
  if (cudaMemsetAsync(workspace, 0, 32, s) != cudaSuccess) {  // status and total start at zero
    cudaGetLastError();
    return PIC_ERR_CUDA;
  }
  if (chunks > 0) {
    izpr_count<<<static_cast<unsigned>(chunks), kThreads, 0, s>>>(symbols, n_symbols, eob, ws.counts);
    izpr_scan<<<1, 1024, 0, s>>>(ws.counts, chunks, ws.base, ws.total);
    izpr_compact<<<static_cast<unsigned>(chunks), kThreads, 0, s>>>(symbols, n_symbols, eob, ws.base,
                                                                    offsets, n_blocks, ws.status);
  }
  if (n_blocks > 0) {
    long long grid = (n_blocks + kThreads / 32 - 1) / (kThreads / 32);
    if (grid > 152 * 16) grid = 152 * 16;
    izpr_expand<<<static_cast<unsigned>(grid), kThreads, 0, s>>>(symbols, eob, offsets, n_blocks,
                                                                 ws.total, coeffs, ws.status);
  }
  if (cudaGetLastError() != cudaSuccess) return PIC_ERR_CUDA;
  return PIC_OK;
}

int pic_izpr_status(const void* workspace, void* stream) {
  if (!workspace) return PIC_ERR_INVALID_ARG;
  int st = 0;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaMemcpyAsync(&st, workspace, sizeof(int), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess) {
    cudaGetLastError();
    return PIC_ERR_CUDA;
  }
  return st == 0 ? PIC_OK : PIC_ERR_INVALID_ARG;
}

}  // extern "C"
