// k_izpr.cu -- inverse ZpR on the GPU (Sec. 3.3, Fig. 2; App. B, Algorithm 1),
// behind the C ABI of include/pic_izpr.h.
//
// Algorithm 1 expands each block from its end-of-block marker offsets, which
// the paper finds beforehand by a stream compaction.  Here:
// 1. izpr_count: eob markers per 4096-symbol chunk (coalesced reads).
// 2. izpr_scan: one CTA, exclusive scan of the chunk counts = index of each
//    chunk's first block; the marker total.
// 3. izpr_expand: persistent CTAs do the compaction and the expansion
//    together, chunk by chunk.  A CTA stages a chunk and the 96 symbols
//    before it in shared memory by cp.async while it works on its previous
//    chunk (a block has at most 64 symbols before its marker, so the marker
//    ending the previous block is in that halo), ranks the chunk's markers
//    with warp ballots (their stream indices are Algorithm 1's offsets), and
//    expands the blocks 8 lanes per block: lane k owns symbols 8k..8k+7 of
//    the block and counts the zigzag positions they cover (1 for a literal,
//    n for the run code of n zeros), a scan over the 8 lanes turns the
//    counts into positions, literals are scattered into a zeroed 64-entry
//    block in shared memory through the zigzag table, and the block leaves
//    as 256 contiguous bytes (two 16-byte stores per lane).
// The stream is read twice (steps 1 and 3); nothing else touches HBM but
// the coefficients and offsets written.
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

// Compaction and expansion in one pass over the stream.  A block holds at
// most 64 symbols before its marker, so the marker that precedes a chunk's
// first block lies within the kHalo symbols before the chunk (or the block
// is malformed).  Persistent CTAs take chunks c, c + grid, ...; each stages
// the halo and the chunk in shared memory by cp.async one chunk ahead
// (double buffer), finds the chunk's markers in stream order (block
// q = base[chunk] + rank), writes their offsets, and expands the chunk's
// blocks straight from shared memory.
constexpr int kHalo = 96;
constexpr int kStageInts = kHalo + kChunk;
// Staged symbol j sits at word j + j / 32: the lanes of a block, which read
// symbols 8 apart, then fall in distinct banks.
constexpr int kStagePadded = kStageInts + kStageInts / 32 + 1;
__device__ __forceinline__ int pad(int j) { return j + (j >> 5); }
constexpr int kExpandSmem = 2 * kStagePadded * 4          // symbols, double buffer
                            + kChunk * 2                  // marker positions (u16)
                            + 4 * (kThreads / 32) * 64 * 4  // one 64-entry block per octet
                            + 64 * 4 + 64 + 16;           // scan scratch, zigzag table, halo marker

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void cp_async4(uint32_t dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_prev() {  // all but the newest group have landed
  asm volatile("cp.async.wait_group 1;" ::: "memory");
}

__global__ void __launch_bounds__(kThreads, 4) izpr_expand(const int32_t* __restrict__ sym,
                                                        long long n, int32_t eob,
                                                        const long long* __restrict__ base,
                                                        const long long* total, long long n_blocks,
                                                        int32_t* __restrict__ coeffs,
                                                        int64_t* __restrict__ offsets, int* status) {
  extern __shared__ __align__(16) unsigned char smem[];
  int* s_sym0 = reinterpret_cast<int*>(smem);
  unsigned short* s_mk = reinterpret_cast<unsigned short*>(smem + 2 * kStagePadded * 4);
  int(*s_blk)[64] = reinterpret_cast<int(*)[64]>(smem + 2 * kStagePadded * 4 + kChunk * 2);
  int* s_scan = reinterpret_cast<int*>(smem + 2 * kStagePadded * 4 + kChunk * 2 +
                                       4 * (kThreads / 32) * 64 * 4);
  unsigned char* s_zz = reinterpret_cast<unsigned char*>(s_scan + 64);  // zigzag table
  int* s_prev = reinterpret_cast<int*>(s_zz + 64);
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const long long n_chunks = (n + kChunk - 1) / kChunk;
  if (t < 64) s_zz[t] = static_cast<unsigned char>(kZigzag.v[t]);
  if (blockIdx.x == 0 && t == 0) {
    if (*total != n_blocks) atomicOr(status, kBadCount);
    if (__ldg(sym + n - 1) != eob) atomicOr(status, kBadCount);  // symbols after the last marker
  }

  // stage chunk c into buffer dst: positions before the stream act as
  // markers (the first block starts at 0); positions past its end hold 0
  // and are never counted
  auto stage = [&](long long c, int* dst) {
    const long long c0 = c * kChunk;
    const uint32_t d = smem_u32(dst);
    for (int j = t; j < kStageInts; j += kThreads) {
      const long long i = c0 - kHalo + j;
      if (i >= 0 && i < n) cp_async4(d + 4 * pad(j), sym + i);
      else dst[pad(j)] = i < 0 ? eob : 0;
    }
  };

  int buf = 0;
  if (blockIdx.x < n_chunks) stage(blockIdx.x, s_sym0);
  cp_async_commit();
  for (long long c = blockIdx.x; c < n_chunks; c += gridDim.x, buf ^= 1) {
    int* s_sym = s_sym0 + buf * kStagePadded;
    if (c + gridDim.x < n_chunks) stage(c + gridDim.x, s_sym0 + (buf ^ 1) * kStagePadded);
    cp_async_commit();
    cp_async_wait_prev();
    __syncthreads();  // chunk c is in s_sym
    const long long c0 = c * kChunk;  // stream index of s_sym[kHalo]

    // markers of the chunk in stream order: warp w scans symbols
    // kHalo + 512 w .. + 511 in 16 steps of 32 (one per lane, conflict-free),
    // ballots give each marker its rank
    constexpr int kSpan = kChunk / (kThreads / 32);
    unsigned mk_mask[kSpan / 32];
    int wcount = 0;
#pragma unroll
    for (int st = 0; st < kSpan / 32; ++st) {
      const int j = kHalo + kSpan * warp + 32 * st + lane;
      mk_mask[st] = __ballot_sync(0xffffffffu, c0 + (j - kHalo) < n && s_sym[pad(j)] == eob);
      wcount += __popc(mk_mask[st]);
    }
    if (lane == 0) s_scan[warp] = wcount;
    __syncthreads();
    int run = 0, tot = 0;
#pragma unroll
    for (int w2 = 0; w2 < kThreads / 32; ++w2) {
      const int v = s_scan[w2];
      run += w2 < warp ? v : 0;
      tot += v;
    }
    const unsigned lt = (1u << lane) - 1u;
#pragma unroll
    for (int st = 0; st < kSpan / 32; ++st) {
      const unsigned m = mk_mask[st];
      if ((m >> lane) & 1u)
        s_mk[run + __popc(m & lt)] = static_cast<unsigned short>(kHalo + kSpan * warp + 32 * st + lane);
      run += __popc(m);
    }
    if (warp == 0) {  // the last marker of the halo, if any
      int last = -1;
#pragma unroll
      for (int h = 0; h < kHalo / 32; ++h) {
        const unsigned m = __ballot_sync(0xffffffffu, s_sym[pad(32 * h + lane)] == eob);
        if (m) last = 32 * h + 31 - __clz(static_cast<int>(m));
      }
      if (lane == 0) *s_prev = last;
    }
    __syncthreads();

    // expansion: 8 lanes per block (an "octet", 4 blocks per warp at a time);
    // lane k of an octet owns symbols 8k .. 8k+7 of its block (a block has at
    // most 64), counts the zigzag positions they cover, and after an
    // exclusive scan over the octet scatters its literals.
    const long long gb0 = base[c];
    const int oct = lane >> 3, k = lane & 7;
    const unsigned omask = 0xffu << (8 * oct);
    int* blk = s_blk[4 * warp + oct];
    for (int q0 = 4 * warp; q0 < tot; q0 += 4 * (kThreads / 32)) {  // warp-uniform trip count
      const int q = q0 + oct;
      const bool has = q < tot;
      int start = 0, end = 0, len = 0;
      bool bad = false;
      if (has) {
        end = s_mk[q];
        const int prev = q == 0 ? *s_prev : s_mk[q - 1];
        start = prev + 1;
        len = end - start;
        bad = prev < 0 || len > 64;
      }
      reinterpret_cast<int4*>(blk)[2 * k] = make_int4(0, 0, 0, 0);
      reinterpret_cast<int4*>(blk)[2 * k + 1] = make_int4(0, 0, 0, 0);
      int sv[8], cnt[8], sum = 0;
      unsigned lit = 0;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int e = 8 * k + i;
        sv[i] = 0;
        cnt[i] = 0;
        if (has && !bad && e < len) {
          sv[i] = s_sym[pad(start + e)];
          const bool run = sv[i] >= eob - 16 && sv[i] < eob;
          cnt[i] = run ? sv[i] - (eob - 17) : 1;  // run of n zeros, or a literal
          if (!run) lit |= 1u << i;
          if (sv[i] > eob) bad = true;
        }
        sum += cnt[i];
      }
      int x = sum;  // inclusive scan over the octet
#pragma unroll
      for (int o = 1; o < 8; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o, 8);
        if (k >= o) x += y;
      }
      const int covered = __shfl_sync(0xffffffffu, x, 7, 8);
      bad = (__ballot_sync(0xffffffffu, bad || covered > 64) & omask) != 0;
      __syncwarp();  // the zeroed buffer is complete
      if (!bad) {
        int pos = x - sum;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          if (lit & (1u << i)) blk[s_zz[pos]] = sv[i];
          pos += cnt[i];
        }
      }
      __syncwarp();
      if (has) {
        if (bad && k == 0) atomicOr(status, kBadBlock);
        const long long gb = gb0 + q;
        if (gb < n_blocks) {
          int4* dst = reinterpret_cast<int4*>(coeffs + gb * 64);
          dst[2 * k] = reinterpret_cast<const int4*>(blk)[2 * k];
          dst[2 * k + 1] = reinterpret_cast<const int4*>(blk)[2 * k + 1];
          if (k == 0) offsets[gb] = c0 - kHalo + end;
        } else if (k == 0) {
          atomicOr(status, kBadCount);
        }
      }
      __syncwarp();
    }
    __syncthreads();  // s_mk, the octet buffers and this symbol buffer are free again
  }
}

__global__ void izpr_flag(int* status, int bits) { atomicOr(status, bits); }

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// Persistent grid of izpr_expand on the current device (resident CTAs over
// all SMs), set up once per device.
int expand_grid(int* grid) {
  constexpr int kMaxDev = 64;
  static int cached[kMaxDev];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDev) {
    cudaGetLastError();
    return PIC_ERR_CUDA;
  }
  if (cached[dev] == 0) {
    int sms = 0, per_sm = 0;
    if (cudaFuncSetAttribute(izpr_expand, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             kExpandSmem) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, izpr_expand, kThreads,
                                                      kExpandSmem) != cudaSuccess ||
        per_sm < 1) {
      cudaGetLastError();
      return PIC_ERR_CUDA;
    }
    cached[dev] = sms * per_sm;
  }
  *grid = cached[dev];
  return PIC_OK;
}

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
    int grid = 0;
    if (expand_grid(&grid) != PIC_OK) return PIC_ERR_CUDA;
    izpr_expand<<<static_cast<unsigned>(chunks < grid ? chunks : grid), kThreads, kExpandSmem, s>>>(
        symbols, n_symbols, eob, ws.base, ws.total, n_blocks, coeffs, offsets, ws.status);
  } else if (n_blocks > 0) {
    izpr_flag<<<1, 1, 0, s>>>(ws.status, kBadCount);  // no symbols, hence no markers
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
