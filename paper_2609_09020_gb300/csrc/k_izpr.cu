// k_izpr.cu -- inverse ZpR on the GPU (Sec. 3.3, Fig. 2; App. B, Algorithm 1),
// behind the C ABI of include/pic_izpr.h.
//
// Algorithm 1 expands each block from its end-of-block marker offsets, which
// the paper finds beforehand by a stream compaction.  Here:
// 1. izpr_count: eob markers per 2048-symbol chunk (16-byte loads), summed
//    over groups of 8 chunks, with each chunk's offset within its group.
// 2. izpr_scan: one CTA, exclusive scan of the group counts; a chunk's
//    first block = its group's base + its offset in the group.
// 3. izpr_expand: persistent CTAs do the compaction and the expansion
//    together, chunk by chunk, as a segmented scan.  Each thread holds 16
//    consecutive symbols of the chunk in registers (loaded while the CTA
//    expanded its previous chunk) and reduces them to (markers, positions
//    covered since its last marker); warp 0 reads the 96 symbols before the
//    chunk (a block has at most 64 symbols before its marker, so the marker
//    ending the previous block is in that halo); a CTA-wide scan gives each
//    thread the block and zigzag position of its first symbol, and each
//    thread walks its symbols as Algorithm 1 walks a block: a literal goes to
//    the next zigzag position, a run code of n zeros skips n positions, a
//    marker closes the block (its stream index is Algorithm 1's offset).  The
//    blocks, assembled in shared memory, leave as whole 256-byte blocks.
// The stream is read twice (steps 1 and 3); nothing else touches HBM but
// the coefficients and offsets written.
#include <cstdint>

#include <cuda_runtime.h>

#include "pic_decode.h"
#include "pic_izpr.h"

namespace pic {
namespace {

constexpr int kThreads = 128;
constexpr int kPerThread = 16;
constexpr int kChunk = kThreads * kPerThread;  // symbols per compaction chunk

enum : int { kBadBlock = 1, kBadCount = 2 };

// Chunks are counted in groups of kGroup (one CTA of kGroup x kThreads
// threads per group), so the scan runs over the groups.
constexpr int kGroup = 8;
// Workspace: status word, marker total, group counts, each chunk's first
// block within its group, group bases.
struct Workspace {
  int* status;
  long long* total;
  int* gcount;
  int* local;
  long long* gbase;
};
__host__ __device__ inline long long n_chunks_of(long long n) { return (n + kChunk - 1) / kChunk; }
__host__ __device__ inline long long n_groups_of(long long n) { return (n_chunks_of(n) + kGroup - 1) / kGroup; }
__host__ __device__ inline long long align16(long long b) { return (b + 15) / 16 * 16; }
__host__ __device__ inline long long ws_bytes(long long n) {
  return 32 + align16(4 * n_groups_of(n)) + align16(4 * n_chunks_of(n)) + 8 * n_groups_of(n);
}
__host__ __device__ inline Workspace ws_view(void* w, long long n) {
  char* p = static_cast<char*>(w);
  const long long g = n_groups_of(n), c = n_chunks_of(n);
  Workspace v;
  v.status = reinterpret_cast<int*>(p);
  v.total = reinterpret_cast<long long*>(p + 16);
  v.gcount = reinterpret_cast<int*>(p + 32);
  v.local = reinterpret_cast<int*>(p + 32 + align16(4 * g));
  v.gbase = reinterpret_cast<long long*>(p + 32 + align16(4 * g) + align16(4 * c));
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

// 16 consecutive symbols from stream index i0 into r; positions past the
// end read as `fill`.  16-byte loads when the stream is 16-byte aligned.
__device__ __forceinline__ void load16(const int32_t* __restrict__ sym, long long n, long long i0,
                                       bool vec, int fill, int (&r)[16]) {
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const long long i = i0 + 4 * q;
    if (vec && i + 3 < n) {
      const int4 v = __ldg(reinterpret_cast<const int4*>(sym + i));
      r[4 * q] = v.x;
      r[4 * q + 1] = v.y;
      r[4 * q + 2] = v.z;
      r[4 * q + 3] = v.w;
    } else {
#pragma unroll
      for (int u = 0; u < 4; ++u) r[4 * q + u] = i + u < n ? __ldg(sym + i + u) : fill;
    }
  }
}

// Markers of the kGroup chunks of group blockIdx.x: thread t counts 16
// symbols of chunk kGroup g + t / kThreads; the group's total, and each
// chunk's count of markers before it within the group.
__global__ void __launch_bounds__(kGroup * kThreads, 2) izpr_count(const int32_t* __restrict__ sym, long long n,
                                                                int32_t eob, long long n_chunks, int* gcount,
                                                                int* local) {
  __shared__ int s_warp[kGroup * kThreads / 32];
  const int t = threadIdx.x, sub = t / kThreads, lane = t & 31;
  const long long c = static_cast<long long>(blockIdx.x) * kGroup + sub;
  const long long i0 = c * kChunk + 16 * (t % kThreads);
  int cnt = 0;
  if (c < n_chunks) {
    int r[16];
    load16(sym, n, i0, (reinterpret_cast<uintptr_t>(sym) & 15u) == 0, eob, r);
#pragma unroll
    for (int k = 0; k < 16; ++k) cnt += (r[k] == eob && i0 + k < n) ? 1 : 0;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, o);
  if (lane == 0) s_warp[t >> 5] = cnt;
  __syncthreads();
  if (t == 0) {
    constexpr int kWarpsPerChunk = kThreads / 32;
    int run = 0;
    for (int q = 0; q < kGroup; ++q) {
      const long long cq = static_cast<long long>(blockIdx.x) * kGroup + q;
      if (cq < n_chunks) local[cq] = run;
      for (int w = 0; w < kWarpsPerChunk; ++w) run += s_warp[q * kWarpsPerChunk + w];
    }
    gcount[blockIdx.x] = run;
  }
}

// One CTA: exclusive scan of the chunk counts into chunk bases; the total.
// Tiles of 8192 counts are staged in shared memory by coalesced loads
// (padded: entry j at j + j / 32); thread t scans entries 8t .. 8t+7.
__global__ void __launch_bounds__(1024) izpr_scan(const int* __restrict__ counts, long long n_chunks,
                                                  long long* base, long long* total) {
  constexpr int kPer = 8, kTileN = 1024 * kPer;
  __shared__ int s_c[kTileN + kTileN / 32];
  __shared__ long long s_w[32];
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  long long carry = 0;
  for (long long t0 = 0; t0 < n_chunks; t0 += kTileN) {
    const long long m = min(static_cast<long long>(kTileN), n_chunks - t0);
    int v[kPer];  // all loads in flight together, then the shared stores
#pragma unroll
    for (int k = 0; k < kPer; ++k) {
      const int j = t + 1024 * k;
      v[k] = j < m ? __ldg(counts + t0 + j) : 0;
    }
#pragma unroll
    for (int k = 0; k < kPer; ++k) {
      const int j = t + 1024 * k;
      s_c[j + (j >> 5)] = v[k];
    }
    __syncthreads();
    long long s = 0;
#pragma unroll
    for (int k = 0; k < kPer; ++k) {
      const int j = kPer * t + k;
      s += s_c[j + (j >> 5)];
    }
    long long x = s;  // inclusive scan: warp, then warp totals
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const long long y = __shfl_up_sync(0xffffffffu, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) s_w[warp] = x;
    __syncthreads();
    if (warp == 0) {
      long long w = s_w[lane];
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const long long y = __shfl_up_sync(0xffffffffu, w, o);
        if (lane >= o) w += y;
      }
      s_w[lane] = w;
    }
    __syncthreads();
    long long run = carry + (warp > 0 ? s_w[warp - 1] : 0) + x - s;
#pragma unroll
    for (int k = 0; k < kPer; ++k) {
      const int j = kPer * t + k;
      if (j < m) base[t0 + j] = run;
      run += s_c[j + (j >> 5)];
    }
    carry += s_w[31];
    __syncthreads();  // s_c and s_w are free again
  }
  if (t == 0) *total = carry;
}

// Compaction and expansion in one pass over the stream, as a segmented scan.
// A block holds at most 64 symbols before its marker, so the marker that
// precedes a chunk's first block lies within the kHalo symbols before the
// chunk (or the block is malformed).  Persistent CTAs take chunks c,
// c + grid, ...; for each:
//  - every thread holds 16 consecutive symbols of the chunk in registers
//    (loaded while the CTA worked on its previous chunk) and reduces them to
//    (markers, positions covered since its last marker);
//  - warp 0 finds the halo's last marker and the positions of the part of
//    the chunk's first block that lies in the halo (they carry in);
//  - a CTA-wide segmented scan of the (markers, positions) pairs gives each
//    thread the block of its first symbol (block q of the chunk = block
//    base[chunk] + q of the stream) and the zigzag position reached in it;
//  - each thread walks its symbols: a literal goes to the block's next
//    zigzag position, a run code of n zeros skips n positions, a marker
//    closes the block (its stream index is Algorithm 1's offset);
//  - the blocks, assembled in shared memory, leave as whole 256-byte blocks
//    in raster order.
// Symbols after the chunk's last marker belong to the next chunk's first
// block; here they land in a spare block slot that is cleared, not written
// out.  A chunk with more than kMaxBlk blocks (only possible with very short
// blocks) is expanded in several passes over its block range.
constexpr int kHalo = 96;                   // 3 symbols per lane of warp 0
constexpr int kMaxBlk = 96;                 // blocks assembled per pass
constexpr int kBlkStride = 68;              // words per block slot: equal raster
                                            // entries of neighbouring blocks
                                            // fall 4 banks apart
constexpr int kExpandSmem = (kMaxBlk + 1) * kBlkStride * 4  // block slots + spare
                            + 64 * 4                        // scan scratch
                            + 64 + 16;                      // zigzag table, halo carry

// Segmented-scan combine: (m1, s1) then (m2, s2) -> markers m1 + m2, and
// the positions covered since the last marker.
struct Seg {
  int m, s;
};
__device__ __forceinline__ Seg seg_cat(Seg a, Seg b) { return Seg{a.m + b.m, b.m > 0 ? b.s : a.s + b.s}; }

__global__ void __launch_bounds__(kThreads, 8) izpr_expand(const int32_t* __restrict__ sym,
                                                        long long n, int32_t eob,
                                                        const long long* __restrict__ gbase,
                                                        const int* __restrict__ local,
                                                        const long long* total, long long n_blocks,
                                                        int32_t* __restrict__ coeffs,
                                                        int64_t* __restrict__ offsets, int* status) {
  extern __shared__ __align__(16) unsigned char smem[];
  int* s_buf = reinterpret_cast<int*>(smem);
  int* s_scan = s_buf + (kMaxBlk + 1) * kBlkStride;
  unsigned char* s_zz = reinterpret_cast<unsigned char*>(s_scan + 64);
  int* s_carry = reinterpret_cast<int*>(s_zz + 64);
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  constexpr int kWarps = kThreads / 32;
  const long long n_chunks = (n + kChunk - 1) / kChunk;
  if (t < 64) s_zz[t] = static_cast<unsigned char>(make_zigzag().v[t]);
  if (blockIdx.x == 0 && t == 0) {
    if (*total != n_blocks) atomicOr(status, kBadCount);
    if (__ldg(sym + n - 1) != eob) atomicOr(status, kBadCount);  // symbols after the last marker
  }
  for (int j = t; j < (kMaxBlk + 1) * kBlkStride / 4; j += kThreads)
    reinterpret_cast<int4*>(s_buf)[j] = make_int4(0, 0, 0, 0);
  const bool vec = (reinterpret_cast<uintptr_t>(sym) & 15u) == 0;
  const uint32_t ueob16 = static_cast<uint32_t>(eob) - 16u;  // first run code
  // Past the end of the stream the symbols read as a literal (eob - 17):
  // never a marker, and only ever in the spare slot.
  const int fill = static_cast<int>(static_cast<uint32_t>(eob) - 17u);

  // The halo of chunk c for warp 0 (lane l: symbols c0 - kHalo + 3 l .. + 2);
  // before the stream they act as markers.
  auto load_halo = [&](long long c, int (&h)[3]) {
    const long long hi = c * kChunk - kHalo + 3 * lane;
#pragma unroll
    for (int u = 0; u < 3; ++u) h[u] = (warp != 0 || hi + u < 0) ? eob : __ldg(sym + hi + u);
  };

  // the next chunk's symbols, halo and first block index, loaded one chunk ahead
  int cur[16], hcur[3];
  long long bcur = 0;
  if (blockIdx.x < n_chunks) {
    load16(sym, n, static_cast<long long>(blockIdx.x) * kChunk + 16 * t, vec, fill, cur);
    load_halo(blockIdx.x, hcur);
    bcur = gbase[blockIdx.x / kGroup] + local[blockIdx.x];
  }
  for (long long c = blockIdx.x; c < n_chunks; c += gridDim.x) {
    const long long c0 = c * kChunk;
    const long long gb0 = bcur;
    int x16[16], h[3];
#pragma unroll
    for (int i = 0; i < 16; ++i) x16[i] = cur[i];
#pragma unroll
    for (int u = 0; u < 3; ++u) h[u] = hcur[u];
    if (c + gridDim.x < n_chunks) {  // next chunk, in flight meanwhile
      load16(sym, n, (c + gridDim.x) * kChunk + 16 * t, vec, fill, cur);
      load_halo(c + gridDim.x, hcur);
      bcur = gbase[(c + gridDim.x) / kGroup] + local[c + gridDim.x];
    }

    // this thread's markers (bit i: symbol i) and positions since its last one
    unsigned mk = 0;
    int s = 0, vmax = x16[0];
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const int x = x16[i];
      const uint32_t d = static_cast<uint32_t>(x) - ueob16;
      const bool m = x == eob;
      mk |= m ? 1u << i : 0u;
      s = m ? 0 : s + (d < 16u ? static_cast<int>(d) + 1 : 1);
      vmax = max(vmax, x);
    }
    bool bad = vmax > eob;
    // warp-inclusive segmented scan
    Seg inc{__popc(mk), s};
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const Seg y{__shfl_up_sync(0xffffffffu, inc.m, o), __shfl_up_sync(0xffffffffu, inc.s, o)};
      if (lane >= o) inc = seg_cat(y, inc);
    }
    if (lane == 31) {
      s_scan[2 * warp] = inc.m;
      s_scan[2 * warp + 1] = inc.s;
    }
    // the halo (warp 0): its last marker, and the positions of the part of
    // the chunk's first block that lies in it
    int halo_pos = 0;
    if (warp == 0) {
      int last = -1;
#pragma unroll
      for (int u = 0; u < 3; ++u)
        if (h[u] == eob) last = 3 * lane + u;
      last = __reduce_max_sync(0xffffffffu, last);
      int sum = 0;
#pragma unroll
      for (int u = 0; u < 3; ++u) {
        if (3 * lane + u <= last || last < 0) h[u] = eob;  // not part of the first block
        const uint32_t d = static_cast<uint32_t>(h[u]) - ueob16;
        sum += h[u] == eob ? 0 : (d < 16u ? static_cast<int>(d) + 1 : 1);
      }
      int x = sum;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
      }
      halo_pos = x - sum;  // zigzag position of this lane's first halo symbol
      // a block with no marker in the halo has more than 64 symbols
      if (lane == 31) *s_carry = last < 0 ? 65 : x;
    }
    __syncthreads();  // warp totals and the halo carry

    // exclusive prefix of this thread: (block of its first symbol, position)
    Seg pre{0, *s_carry};
    int tot = 0;
#pragma unroll
    for (int w2 = 0; w2 < kWarps; ++w2) {
      const Seg v{s_scan[2 * w2], s_scan[2 * w2 + 1]};
      if (w2 < warp) pre = seg_cat(pre, v);
      tot += v.m;  // blocks of this chunk
    }
    {
      const Seg y{__shfl_up_sync(0xffffffffu, inc.m, 1), __shfl_up_sync(0xffffffffu, inc.s, 1)};
      if (lane > 0) pre = seg_cat(pre, y);
    }
    // offsets (Algorithm 1): the stream index of each marker
    {
      int q = pre.m;
      for (unsigned b = mk; b; b &= b - 1u, ++q) {
        const long long gb = gb0 + q;
        if (gb < n_blocks) offsets[gb] = c0 + 16 * t + (__ffs(b) - 1);
        else atomicOr(status, kBadCount);
      }
    }

    // expansion, kMaxBlk blocks of the chunk per pass; in a pass the blocks
    // outside it (and the next chunk's first block) go to the spare slot
    for (int p0 = 0; p0 < tot; p0 += kMaxBlk) {
      const int p1 = min(tot, p0 + kMaxBlk);
      const bool one_pass = tot <= kMaxBlk;  // then q - p0 never leaves [0, kMaxBlk]
      if (p0 == 0 && warp == 0) {  // the first block's literals from the halo
#pragma unroll
        for (int u = 0; u < 3; ++u) {
          const uint32_t d = static_cast<uint32_t>(h[u]) - ueob16;
          if (h[u] != eob && d > 16u && halo_pos < 64) s_buf[s_zz[halo_pos]] = h[u];
          halo_pos += h[u] == eob ? 0 : (d < 16u ? static_cast<int>(d) + 1 : 1);
        }
      }
      int q = pre.m, pos = pre.s;
      auto slot = [&](int qq) {
        return one_pass ? qq * kBlkStride : ((qq >= p0 && qq < p1) ? qq - p0 : kMaxBlk) * kBlkStride;
      };
      int qb = slot(q);
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const int x = x16[i];
        const uint32_t d = static_cast<uint32_t>(x) - ueob16;  // < 16: run code, 16: marker
        const int zz = s_zz[pos & 63];
        if (d > 16u) s_buf[qb + zz] = x;  // a literal (or a malformed value)
        if (d == 16u) {
          if (pos > 64) bad = true;
          ++q;
          pos = 0;
          qb = slot(q);
        } else {
          pos += d < 16u ? static_cast<int>(d) + 1 : 1;
        }
      }
      __syncthreads();  // the pass's blocks are assembled
      // copy-out: two blocks per warp instruction, 16 bytes per lane; every
      // slot used (the spare one too) is cleared for the next pass
      const int last_slot = one_pass ? p1 - p0 : kMaxBlk;
      for (int b = 2 * warp + (lane >> 4); b <= last_slot; b += 2 * kWarps) {
        int4* src = reinterpret_cast<int4*>(s_buf + b * kBlkStride) + (lane & 15);
        const int4 v = *src;
        *src = make_int4(0, 0, 0, 0);
        const long long gb = gb0 + p0 + b;
        if (b < p1 - p0 && gb < n_blocks) reinterpret_cast<int4*>(coeffs + gb * 64)[lane & 15] = v;
      }
      __syncthreads();  // the slots are clear again
    }
    if (bad) atomicOr(status, kBadBlock);
    __syncthreads();  // the scan scratch and the halo carry are free again
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
    const long long groups = n_groups_of(n_symbols);
    izpr_count<<<static_cast<unsigned>(groups), kGroup * kThreads, 0, s>>>(symbols, n_symbols, eob, chunks,
                                                                           ws.gcount, ws.local);
    izpr_scan<<<1, 1024, 0, s>>>(ws.gcount, groups, ws.gbase, ws.total);
    int grid = 0;
    if (expand_grid(&grid) != PIC_OK) return PIC_ERR_CUDA;
    izpr_expand<<<static_cast<unsigned>(chunks < grid ? chunks : grid), kThreads, kExpandSmem, s>>>(
        symbols, n_symbols, eob, ws.gbase, ws.local, ws.total, n_blocks, coeffs, offsets, ws.status);
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
