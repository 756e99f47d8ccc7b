// k_huffman.cu -- Huffman decoding of B image-specific streams on the GPU
// (include/pic_huffman.h; Sec. 3.3 and Sec. 4.1 of the paper, which adapts
// GPUHD, Weissenberger & Schmidt 2018: self-synchronising parallel decoding).
//
// 1. huff_lut (one CTA per image): the stored table -- values and lengths in
//    canonical order -- is the run-length code of the 2^p-entry lookup table:
//    symbol k covers 2^(p - len_k) consecutive entries.  Expanding the runs
//    gives the table (16-bit entry = length << 12 | k, the symbol's row in
//    the stored table, whose value is read only when it is written out), so
//    one lookup of the next p bits decodes a symbol.  Kraft's inequality is
//    checked here.
// 2. huff_decode (one cooperative launch; every CTA resident, grid-wide
//    barriers between the phases):
//    a. each thread decodes its 256-bit subsequences speculatively from their
//       first bit, which may lie inside a codeword, until it passes the
//       subsequence's end; it records the first codeword boundary at or
//       after the end (the exit) and the number of codewords started;
//    b. synchronisation passes: a subsequence whose start differs from its
//       predecessor's exit is decoded again from that exit.  Prefix codes
//       resynchronise within a few codewords, so the passes stop changing
//       after one or two; pass i has made subsequence i exact, and after 64
//       passes without convergence the status word says so;
//    c. an exclusive scan of the codeword counts gives every subsequence's
//       output position (each image's must equal its symbol offset);
//    d. every subsequence is decoded from its final start, writing values.
// Each CTA stages its images' lookup tables and, per pass, the stream words
// of its 256 subsequences in shared memory.  Each thread keeps a 64-bit
// window of the stream in registers and reloads one word when its position
// crosses a word boundary (codes are at most 12 bits, so at most one word per
// codeword).  The counting decodes of a and b use a pair table per image (the
// lengths of the first two codewords of every p-bit window, when both lie
// inside it), so one lookup advances over up to two codewords.  The final
// decode d writes through per-warp staging rows, 16 symbols per thread per
// round, so that each warp store writes two whole 64-byte runs.
#include <cstdint>

#include <cooperative_groups.h>
#include <cuda_runtime.h>

#include "pic_decode.h"
#include "pic_huffman.h"

namespace cg = cooperative_groups;

namespace {

constexpr int kQ = PIC_HUFF_WORDS_PER_SUBSEQ;  // words per subsequence
constexpr int kS = 32 * kQ;                     // bits per subsequence
constexpr int kThreads = 256;
constexpr int kMaxPasses = 64;
constexpr int kMaxTable = 4096;
constexpr int kMaxGrid = 8192;
constexpr int kWbuf = kThreads * kQ + 2;  // stream words of one pass of 256 subsequences
constexpr int kRound = 16;                // symbols a thread decodes between two warp stores
constexpr int kRow = kRound + 1;          // staging row (padded against bank conflicts)
constexpr int kStageInts = kThreads * kRow;
enum : int { kBadCode = 1, kBadCount = 2, kNoSync = 4, kBadTable = 8 };

struct Ws {
  int* status;           // [4]
  int* changed;          // [kMaxPasses]
  long long* block_sum;  // [kMaxGrid]
  uint16_t* lut;         // [B][2^p]
  long long* exit0;      // [n_sub]
  long long* exit1;      // [n_sub]
  long long* start;      // [n_sub]
  long long* off;        // [n_sub]
  int* cnt;              // [n_sub]
};

long long ws_size(long long n_sub, int B, int p) {
  long long b = 16 + kMaxPasses * 4 + kMaxGrid * 8;
  b += (static_cast<long long>(B) << p) * 2;
  b = (b + 15) / 16 * 16;
  b += n_sub * (8 * 4 + 4);
  return (b + 15) / 16 * 16;
}

__host__ __device__ inline Ws ws_view(void* w, long long n_sub, int B, int p) {
  char* c = static_cast<char*>(w);
  Ws v;
  v.status = reinterpret_cast<int*>(c);
  v.changed = reinterpret_cast<int*>(c + 16);
  v.block_sum = reinterpret_cast<long long*>(c + 16 + kMaxPasses * 4);
  v.lut = reinterpret_cast<uint16_t*>(c + 16 + kMaxPasses * 4 + kMaxGrid * 8);
  long long o = 16 + kMaxPasses * 4 + kMaxGrid * 8 + (static_cast<long long>(B) << p) * 2;
  o = (o + 15) / 16 * 16;
  v.exit0 = reinterpret_cast<long long*>(c + o);
  v.exit1 = v.exit0 + n_sub;
  v.start = v.exit1 + n_sub;
  v.off = v.start + n_sub;
  v.cnt = reinterpret_cast<int*>(v.off + n_sub);
  return v;
}

// ---------------------------------------------------------------- 1. tables
__global__ void __launch_bounds__(kThreads)
    huff_lut(const int32_t* __restrict__ tab_len, int max_table, int p, uint16_t* lut, int* status) {
  __shared__ int s_start[kMaxTable + 1];
  __shared__ uint16_t s_entry[kMaxTable];
  __shared__ int s_warp[kThreads / 32];
  __shared__ int s_m;
  const int b = blockIdx.x, t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const int32_t* tl = tab_len + static_cast<long long>(b) * max_table;
  // the table ends at its first zero length
  if (t == 0) s_m = max_table;
  __syncthreads();
  for (int k = t; k < max_table; k += blockDim.x)
    if (tl[k] == 0) atomicMin(&s_m, k);
  __syncthreads();
  const int m = s_m;
  // run sizes 2^(p - len) scanned into run starts, 256 entries at a time
  bool bad = false;
  int carry = 0;
  for (int k0 = 0; k0 < m; k0 += kThreads) {
    const int k = k0 + t;
    int run = 0;
    if (k < m) {
      const int l = tl[k];
      if (l < 1 || l > p) bad = true;
      else run = 1 << (p - l);
      s_entry[k] = static_cast<uint16_t>((l << 12) | k);  // the value is tab_value[k]
    }
    int x = run;  // inclusive warp scan, then across the warps
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) s_warp[warp] = x;
    __syncthreads();
    int before = 0, total = 0;
    for (int i = 0; i < kThreads / 32; ++i) {
      before += i < warp ? s_warp[i] : 0;
      total += s_warp[i];
    }
    if (k < m) s_start[k] = min(carry + before + x - run, 1 << p);
    carry = min(carry + total, (1 << p) + 1);  // capped: runs may sum past 2^p only in bad tables
    __syncthreads();
  }
  bad = __syncthreads_or(bad) || carry > (1 << p);  // a bad length, or Kraft's inequality violated
  if (t == 0) {
    s_start[m] = bad ? 0 : carry;
    if (bad) atomicOr(status, kBadTable);
  }
  __syncthreads();
  const int fill = s_start[m];  // a bad table decodes nothing: every entry "no codeword"
  uint16_t* out = lut + (static_cast<long long>(b) << p);
  // every entry finds its run by binary search over the run starts
  for (int i = t; i < (1 << p); i += blockDim.x) {
    uint16_t e = 0;  // no codeword
    if (i < fill) {
      int lo = 0, hi = m - 1;  // last k with s_start[k] <= i
      while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (s_start[mid] <= i) lo = mid;
        else hi = mid - 1;
      }
      e = s_entry[lo];
    }
    out[i] = e;
  }
}

// --------------------------------------------------------------- 2. decode
struct DecodeParams {
  const uint32_t* words;
  long long n_words;
  const long long* word_off;
  const long long* n_bits;
  int B;
  int p;
  const long long* sym_off;
  const int32_t* tab_value;  // [B][max_table]: a table entry's low 12 bits index its row
  int max_table;
  int32_t* out;
  Ws ws;
  long long n_sub;
  long long per_block;  // subsequences per CTA, a multiple of kThreads
};

__device__ __forceinline__ int image_of(const DecodeParams& P, long long word) {
  int lo = 0, hi = P.B - 1;  // last b with word_off[b] <= word
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (__ldg(P.word_off + mid) <= word) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

// The counting loop of decode_span_s, with (PAIR) or without the pair table.
template <bool PAIR>
__device__ __forceinline__ int decode_span_loop(const uint32_t* sw, int lpos, int lke, const uint16_t* lut,
                                                const uint8_t* lut2, int p, int* count, bool* bad) {
  int c = 0;
  int li = lpos >> 5;
  uint32_t hi = sw[li], lo = sw[li + 1];
  const int shr = 32 - p;
  while (lpos < lke) {
    const int wi = lpos >> 5;
    if (wi != li) {  // crossed into the next word (a step covers at most p <= 12 bits)
      li = wi;
      hi = lo;
      lo = sw[li + 1];
    }
    const uint32_t w = __funnelshift_l(lo, hi, lpos & 31) >> shr;
    if constexpr (PAIR) {
      const uint32_t e2 = lut2[w];
      int l1 = static_cast<int>(e2 & 15u);
      const int l2 = static_cast<int>(e2 >> 4);
      if (l1 == 0) {
        *bad = true;
        l1 = 1;
      }
      const bool two = l2 != 0 && lpos + l1 < lke;
      c += two ? 2 : 1;
      lpos += two ? l1 + l2 : l1;
    } else {
      int len = static_cast<int>(lut[w] >> 12);
      if (len == 0) {
        *bad = true;
        len = 1;
      }
      ++c;
      lpos += len;
    }
  }
  *count = c;
  return lpos;
}

// Counts the codewords from bit `lpos` of the words staged in shared memory
// (bit 0 = the top bit of sw[0]) while lpos < lke; returns the position
// after the last codeword.  *bad is raised on a bit pattern that is no
// codeword.  The next p bits come from one funnel shift of the two current
// words.  With a pair table (lut2: the lengths of the first codeword of each
// p-bit window and of the second one when it lies inside the same window),
// one lookup advances over up to two codewords.
__device__ __forceinline__ int decode_span_s(const uint32_t* sw, int lpos, int lke, const uint16_t* lut,
                                             const uint8_t* lut2, int p, int* count, bool* bad) {
  if (lpos >= lke) {
    *count = 0;
    return lpos;
  }
  return lut2 ? decode_span_loop<true>(sw, lpos, lke, lut, lut2, p, count, bad)
              : decode_span_loop<false>(sw, lpos, lke, lut, lut2, p, count, bad);
}

// decode_span_s for subsequence positions of image b: pos (bits from the
// image's first word wbase) <-> staged position (bits from word w0).
__device__ __forceinline__ long long decode_at(const uint32_t* sw, long long w0, long long wbase, long long pos,
                                               long long ke, const uint16_t* lut, const uint8_t* lut2, int p,
                                               int* count, bool* bad) {
  if (pos >= ke) {
    *count = 0;
    return pos;
  }
  const long long shift = (wbase - w0) * 32;  // staged bit = image bit + shift (>= 0 here)
  const int lp = decode_span_s(sw, static_cast<int>(pos + shift), static_cast<int>(ke + shift), lut, lut2, p,
                               count, bad);
  return lp - shift;
}

__device__ long long block_sum_ll(long long v, long long* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  long long t = 0;
  for (int i = 0; i < kThreads / 32; ++i) t += red[i];
  return t;
}

__global__ void __launch_bounds__(kThreads) huff_decode(const DecodeParams P) {
  cg::grid_group grid = cg::this_grid();
  __shared__ long long red[kThreads / 32];
  __shared__ long long scan[kThreads];
  extern __shared__ __align__(16) uint32_t s_dyn[];
  uint16_t* s_lut = reinterpret_cast<uint16_t*>(s_dyn);  // tables of the first and last image of the range
  const Ws& ws = P.ws;
  const long long per_block = P.per_block;
  const long long k_begin = static_cast<long long>(blockIdx.x) * per_block;
  const long long k_end = min(k_begin + per_block, P.n_sub);
  bool bad = false;
  // every lookup is a dependent load in a decode chain: the CTA's images'
  // tables go to shared memory (images between the first and the last of
  // the range, which only tiny streams produce, read theirs from global)
  const int tsize = 1 << P.p;
  const int b_first = k_begin < k_end ? image_of(P, k_begin * kQ) : 0;
  const int b_last = k_begin < k_end ? image_of(P, (k_end - 1) * kQ) : 0;
  for (int i = threadIdx.x; i < tsize; i += blockDim.x) {
    s_lut[i] = ws.lut[(static_cast<long long>(b_first) << P.p) + i];
    s_lut[tsize + i] = ws.lut[(static_cast<long long>(b_last) << P.p) + i];
  }
  __syncthreads();
  auto lut_of = [&](int b) -> const uint16_t* {
    return b == b_first ? s_lut : (b == b_last ? s_lut + tsize : ws.lut + (static_cast<long long>(b) << P.p));
  };
  // each pass of 256 subsequences first stages its stream words (coalesced),
  // so that no global load sits inside a decode chain
  uint32_t* s_words = reinterpret_cast<uint32_t*>(s_lut + 2 * tsize);
  int* s_stage = reinterpret_cast<int*>(s_words + kWbuf);
  // the pair tables of the two images: first codeword's length | the
  // second's << 4 (0 when it does not lie inside the same p-bit window)
  uint8_t* s_lut2 = reinterpret_cast<uint8_t*>(s_stage + kStageInts);
  for (int i = threadIdx.x; i < 2 * tsize; i += blockDim.x) {
    const uint16_t* L = s_lut + (i >= tsize ? tsize : 0);
    const int w = i & (tsize - 1);
    const int l1 = static_cast<int>(L[w] >> 12);
    int l2 = 0;
    if (l1 > 0 && l1 < P.p) {
      const int l = static_cast<int>(L[(w << l1) & (tsize - 1)] >> 12);
      if (l > 0 && l <= P.p - l1) l2 = l;
    }
    s_lut2[i] = static_cast<uint8_t>(l1 | (l2 << 4));
  }
  __syncthreads();
  auto lut2_of = [&](int b) -> const uint8_t* {
    return b == b_first ? s_lut2 : (b == b_last ? s_lut2 + tsize : nullptr);
  };
  auto stage_words = [&](long long k0) {
    const long long w0 = k0 * kQ;
    __syncthreads();
    for (int i = threadIdx.x; i < kWbuf; i += blockDim.x)
      s_words[i] = w0 + i < P.n_words ? __ldg(P.words + w0 + i) : 0u;
    __syncthreads();
  };

  // a. speculative decode of every subsequence from its first bit
  for (long long k0 = k_begin; k0 < k_end; k0 += kThreads) {
    stage_words(k0);
    const long long k = k0 + threadIdx.x;
    if (k >= k_end) continue;
    const int b = image_of(P, k * kQ);
    const long long wbase = __ldg(P.word_off + b), nb = __ldg(P.n_bits + b);
    const long long ks = (k * kQ - wbase) * 32, ke = min(ks + kS, nb);
    int c = 0;
    bool junk = false;
    const long long ex = decode_at(s_words, k0 * kQ, wbase, ks, ke, lut_of(b), lut2_of(b), P.p, &c, &junk);
    ws.exit0[k] = ex;
    ws.start[k] = ks;
    ws.cnt[k] = c;
  }
  grid.sync();

  // b. synchronisation passes (exits double-buffered)
  int pass = 0;
  bool stable = false;
  for (; pass < kMaxPasses; ++pass) {
    const long long* ex_in = (pass & 1) ? ws.exit1 : ws.exit0;
    long long* ex_out = (pass & 1) ? ws.exit0 : ws.exit1;
    long long ch = 0;
    for (long long k0 = k_begin; k0 < k_end; k0 += kThreads) {
      const long long k = k0 + threadIdx.x;
      int b = 0;
      long long wbase = 0, nb = 0, ks = 0, st = 0;
      bool redo = false;
      if (k < k_end) {
        b = image_of(P, k * kQ);
        wbase = __ldg(P.word_off + b);
        nb = __ldg(P.n_bits + b);
        ks = (k * kQ - wbase) * 32;
        st = ks == 0 || ks >= nb ? ws.start[k] : ex_in[k - 1];
        redo = st != ws.start[k];
        if (!redo) ex_out[k] = ex_in[k];
      }
      if (!__syncthreads_or(redo)) continue;  // nothing to redo in this pass of the CTA
      stage_words(k0);
      if (redo) {
        int c = 0;
        bool junk = false;
        ex_out[k] = decode_at(s_words, k0 * kQ, wbase, st, min(ks + kS, nb), lut_of(b), lut2_of(b), P.p, &c,
                              &junk);
        ws.start[k] = st;
        ws.cnt[k] = c;
        ++ch;
      }
    }
    ch = block_sum_ll(ch, red);
    if (threadIdx.x == 0 && ch) atomicAdd(ws.changed + pass, 1);
    grid.sync();
    if (*reinterpret_cast<volatile int*>(ws.changed + pass) == 0) {
      stable = true;
      break;
    }
  }
  if (!stable && blockIdx.x == 0 && threadIdx.x == 0) atomicOr(ws.status, kNoSync);

  // c. output positions: exclusive scan of the counts in subsequence order
  long long mine = 0;
  for (long long k = k_begin + threadIdx.x; k < k_end; k += blockDim.x) mine += ws.cnt[k];
  mine = block_sum_ll(mine, red);
  if (threadIdx.x == 0) ws.block_sum[blockIdx.x] = mine;
  grid.sync();
  long long base = 0;
  for (int j = threadIdx.x; j < static_cast<int>(blockIdx.x); j += blockDim.x) base += ws.block_sum[j];
  base = block_sum_ll(base, red);
  long long carry = base;
  for (long long k0 = k_begin; k0 < k_end; k0 += blockDim.x) {
    const long long k = k0 + threadIdx.x;
    const long long v = k < k_end ? ws.cnt[k] : 0;
    const int ln = threadIdx.x & 31, wp = threadIdx.x >> 5;
    long long x = v;  // inclusive scan: warp shuffles, then the warp totals
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const long long y = __shfl_up_sync(0xffffffffu, x, o);
      if (ln >= o) x += y;
    }
    __syncthreads();  // scan[] of the previous pass has been read
    if (ln == 31) scan[wp] = x;
    __syncthreads();
    long long before = 0, all = 0;
#pragma unroll
    for (int i = 0; i < kThreads / 32; ++i) {
      before += i < wp ? scan[i] : 0;
      all += scan[i];
    }
    if (k < k_end) ws.off[k] = carry + before + x - v;
    carry += all;
  }
  if (blockIdx.x == gridDim.x - 1 && threadIdx.x == 0 && carry != __ldg(P.sym_off + P.B))
    atomicOr(ws.status, kBadCount);
  __syncthreads();

  // d. final decode from the synchronised starts.  Each thread decodes its
  // subsequence in rounds of up to kRound symbols into its row of a per-warp
  // shared buffer; the warp then stores two threads' rows per instruction
  // (lanes 0-15 and 16-31: two 64-byte runs) instead of 32 scattered words.
  int* wbuf = s_stage + (threadIdx.x >> 5) * 32 * kRow;
  const int lane = threadIdx.x & 31;
  for (long long k0 = k_begin; k0 < k_end; k0 += kThreads) {
    stage_words(k0);
    const long long k = k0 + threadIdx.x;
    int lpos = 0, lke = 0, li = 0;
    uint32_t hi = 0, lo = 0;
    long long o = 0, room = 0, shift = 0, nb = 0, ks = 0;
    const uint16_t* lut = s_lut;
    const int32_t* vals = P.tab_value;
    bool more = false;
    if (k < k_end) {
      const int b = image_of(P, k * kQ);
      const long long wbase = __ldg(P.word_off + b);
      nb = __ldg(P.n_bits + b);
      ks = (k * kQ - wbase) * 32;
      o = ws.off[k];
      const long long img_end = __ldg(P.sym_off + b + 1);
      if (ks == 0 && o != __ldg(P.sym_off + b)) atomicOr(ws.status, kBadCount);
      room = o < img_end ? img_end - o : 0;
      shift = (wbase - k0 * kQ) * 32;
      const long long st = ws.start[k], ke = min(ks + kS, nb);
      lpos = static_cast<int>(st + shift);
      lke = static_cast<int>(ke + shift);
      lut = lut_of(b);
      vals = P.tab_value + static_cast<long long>(b) * P.max_table;
      more = ks < nb && st < ke;
      if (more) {
        li = lpos >> 5;
        hi = s_words[li];
        lo = s_words[li + 1];
      }
    }
    const int shr = 32 - P.p;
    long long done = 0;
    while (__any_sync(0xffffffffu, more)) {
      int n = 0;
      while (more && n < kRound) {
        const int wi = lpos >> 5;
        if (wi != li) {
          li = wi;
          hi = lo;
          lo = s_words[li + 1];
        }
        const uint32_t e = lut[__funnelshift_l(lo, hi, lpos & 31) >> shr];
        int len = static_cast<int>(e >> 12);
        if (len == 0) {
          bad = true;
          len = 1;
        }
        wbuf[lane * kRow + n] = __ldg(vals + (e & 0xFFFu));  // off the decode chain
        ++n;
        lpos += len;
        more = lpos < lke;
      }
      __syncwarp();
      // this thread's output run: cap values at o + done.  Lanes hold
      // consecutive subsequences, so o + done never falls below lane 0's and
      // exceeds it by less than 2^13 (32 subsequences of at most 256
      // codewords): one shuffle per row carries (offset from lane 0, cap).
      const long long left = room - done;  // symbols this thread may still write
      const int cap = static_cast<int>(min(static_cast<long long>(n), max(left, 0LL)));
      const long long at0 = __shfl_sync(0xffffffffu, o + done, 0);
      const unsigned packed = (static_cast<unsigned>(o + done - at0) << 5) | static_cast<unsigned>(cap);
#pragma unroll 4
      for (int j = 0; j < 16; ++j) {
        const int src = 2 * j + (lane >> 4), i = lane & 15;
        const unsigned pk = __shfl_sync(0xffffffffu, packed, src);
        if (i < static_cast<int>(pk & 31u)) P.out[at0 + (pk >> 5) + i] = wbuf[src * kRow + i];
      }
      done += n;
      __syncwarp();
    }
    if (k < k_end && ks < nb) {
      if (done > room) atomicOr(ws.status, kBadCount);
      if (ks + kS >= nb && lpos - shift != nb) atomicOr(ws.status, kBadCode);  // the last codeword overruns
    }
  }
  if (bad) atomicOr(ws.status, kBadCode);
}

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// Resident CTAs of huff_decode on the current device with `smem` bytes of
// lookup tables each (the cooperative grid), per device and precision.
int decode_grid(int p, size_t smem, int* grid) {
  constexpr int kMaxDev = 64;
  static int cached[kMaxDev][PIC_HUFF_MAX_PRECISION + 1];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDev) {
    cudaGetLastError();
    return PIC_ERR_CUDA;
  }
  if (cached[dev][p] == 0) {
    int coop = 0, sms = 0, per_sm = 0;
    // the attribute is the function's, for every precision: set it to the largest
    constexpr int kMaxSmem = (3 * 2 << PIC_HUFF_MAX_PRECISION) + (kWbuf + kStageInts) * 4;
    if (cudaFuncSetAttribute(huff_decode, cudaFuncAttributeMaxDynamicSharedMemorySize, kMaxSmem) !=
            cudaSuccess ||
        cudaDeviceGetAttribute(&coop, cudaDevAttrCooperativeLaunch, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, huff_decode, kThreads, smem) != cudaSuccess) {
      cudaGetLastError();
      return PIC_ERR_CUDA;
    }
    if (!coop || per_sm < 1) return PIC_ERR_UNSUPPORTED;
    cached[dev][p] = sms * per_sm < kMaxGrid ? sms * per_sm : kMaxGrid;
  }
  *grid = cached[dev][p];
  return PIC_OK;
}

}  // namespace

extern "C" {

int64_t pic_huffman_workspace_bytes(int64_t n_words, int B, int p) {
  if (n_words < 0 || n_words % kQ != 0 || B < 1 || p < 1 || p > PIC_HUFF_MAX_PRECISION) return -1;
  return ws_size(n_words / kQ, B, p);
}

int pic_huffman_decode(const uint32_t* words, int64_t n_words, const int64_t* word_off,
                       const int64_t* n_bits, int B, const int32_t* tab_value, const int32_t* tab_len,
                       int max_table, int p, const int64_t* sym_off, int32_t* out, void* workspace,
                       size_t workspace_bytes, void* stream) {
  if (n_words < 1 || n_words % kQ != 0 || B < 1 || B > 65536 || p < 1 || p > PIC_HUFF_MAX_PRECISION ||
      max_table < 1 || max_table > kMaxTable)
    return PIC_ERR_INVALID_ARG;
  if (!words || !word_off || !n_bits || !tab_value || !tab_len || !sym_off || !out || !workspace ||
      !aligned(words, 16) || !aligned(workspace, 16) || !aligned(word_off, 8) || !aligned(n_bits, 8) ||
      !aligned(sym_off, 8) || !aligned(tab_value, 4) || !aligned(tab_len, 4) || !aligned(out, 4))
    return PIC_ERR_INVALID_ARG;
  const long long n_sub = n_words / kQ;
  if (static_cast<long long>(workspace_bytes) < ws_size(n_sub, B, p)) return PIC_ERR_INVALID_ARG;
  // 2 tables + the pass's words + the output staging rows + 2 pair tables
  const size_t lut_smem = (sizeof(uint16_t) * 2 << p) + (kWbuf + kStageInts) * sizeof(uint32_t) + (2 << p);
  int grid = 0;
  int rc = decode_grid(p, lut_smem, &grid);
  if (rc != PIC_OK) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  DecodeParams P{};
  P.words = words;
  P.n_words = n_words;
  P.word_off = reinterpret_cast<const long long*>(word_off);
  P.n_bits = reinterpret_cast<const long long*>(n_bits);
  P.B = B;
  P.p = p;
  P.sym_off = reinterpret_cast<const long long*>(sym_off);
  P.tab_value = tab_value;
  P.max_table = max_table;
  P.out = out;
  P.ws = ws_view(workspace, n_sub, B, p);
  P.n_sub = n_sub;
  // whole passes of kThreads subsequences per CTA (no thread idles in a pass)
  const long long passes = (n_sub + static_cast<long long>(grid) * kThreads - 1) /
                           (static_cast<long long>(grid) * kThreads);
  P.per_block = passes * kThreads;
  if (cudaMemsetAsync(workspace, 0, 16 + kMaxPasses * 4, s) != cudaSuccess) {  // status, pass counters
    cudaGetLastError();
    return PIC_ERR_CUDA;
  }
  huff_lut<<<B, kThreads, 0, s>>>(tab_len, max_table, p, P.ws.lut, P.ws.status);
  const long long g = (n_sub + P.per_block - 1) / P.per_block;
  void* args[] = {&P};
  if (cudaLaunchCooperativeKernel(reinterpret_cast<const void*>(huff_decode), dim3(static_cast<unsigned>(g)),
                                  dim3(kThreads), args, lut_smem, s) != cudaSuccess) {
    cudaGetLastError();
    return PIC_ERR_CUDA;
  }
  if (cudaGetLastError() != cudaSuccess) return PIC_ERR_CUDA;
  return PIC_OK;
}

int pic_huffman_status(const void* workspace, void* stream) {
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
