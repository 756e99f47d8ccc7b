// k_tc.cuh -- the tensor-core decode kernel template (PIC_PREC_FP16_TC),
// included by k_tc.cu (int32 latent symbols) and k_tc_f32lat.cu (fp32
// latents); the two instantiation sets compile in parallel.
//
// The synthesis MLP g_s (Sec. 4.1) runs as a chain of tcgen05 MMAs with the
// accumulators in tensor memory (TMEM); dequantisation, bilinear upsampling
// and concatenation of the pyramid levels (Sec. 3.1, Eq. 1) produce the first
// layer's operand directly in shared memory, and the clamped RGB leaves the
// last accumulator straight for global memory.  Nothing between the latents
// and the RGB planes touches HBM.
//
// Precision: weights are fp16 (used exactly as given).  Every activation
// operand a (feature or hidden value, fp32) is split into two fp16 terms
//   a_hi = a rounded toward zero to fp16,
//   a_lo = fp16(a - a_hi)      (a - a_hi is exact in fp32 and has a's sign,
//                               so ReLU may be applied to each term alone),
// and each layer computes W a_hi + W a_lo with fp32 accumulation, so the
// products carry ~22 significant bits instead of fp16's 11.
//
// Variant with the lo term in fp8 (LO8, PIC_PREC_FP16_TC_LO8; ReLU nets with
// the output layer on the tensor cores): the hidden activations are kept
// scaled by S = 2^6 -- the first layer's weights and every bias carry S
// (exact, a power of two), ReLU commutes with it, and only the three outputs
// are divided by S.  A hidden operand is a_hi = RZ_fp16(S h) against the
// fp16 weights W plus a_lo = RN_e4m3(S h - a_hi) against an e4m3 copy of W
// (kind::f8f6f4, K = 32 per instruction): half the lo MMAs and a quarter of
// the lo operand's tensor memory, ~15 significant bits per product (S h -
// a_hi is about 2^-11 S h, inside e4m3's range).  S |h| must stay below
// fp16's 65504, i.e. |h| < 1024.
//
// Operands of one 128-pixel tile (row r = pixel r = TMEM lane r; LO8: hidden
// A = [h_hi | h_lo] with h_lo in N/4 columns of four e4m3 each, and the lo
// half of B the e4m3 copy of W_k, in its own shared tile):
//   layer 0  A1 = [f_hi | f_lo | 1 | 0..]  smem, K1 = round16(2 D0 + 1); the bias
//            B1 = [W_0  | W_0  | b_0 | 0..] b_0 rides along as the constant-1 column
//   hidden   A  = [h_hi | h_lo]            TMEM, N/2 + N/2 columns (2 fp16 per column)
//            B  = [W_k | b_k 0..0]          smem; W_k serves the hi and the lo half,
//                                           b_k meets a shared constant tile [1 0..0]
//   output   the same with W_out, b_out padded to 16 rows -- or, for narrow
//            or deep nets (Net::OUTCC), on the CUDA cores in fp32 inside the
//            last hidden layer's epilogue, which saves an MMA round trip
//
// CTA organisation (one CTA per SM, persistent over a contiguous tile range):
//   warps 0 .. 4*NWG-1 : NWG warpgroups; group w owns every NWG-th tile of the
//                        range, TMEM columns [2Nw, 2Nw + 2N) (accumulator,
//                        then operand A) and shared buffers (A1, column
//                        buffer).  Thread r of the group decodes pixel r.
//                        The features of the group's next tile are computed
//                        while the tensor core runs the current tile's
//                        second layer, and handed over once the current
//                        accumulator has been read.
//   warps 4*NWG + w    : group w's issuing warp (together one warpgroup, which
//                        gives registers to the decoders): waits, issues, commits.
// Handshakes are mbarriers; every wait is bounded (on timeout the kernel
// raises the handle's status word, skips the rest and still frees TMEM).
//
// Latent staging.  Each decoding thread loads its share of the next tile's
// coarse-level source rows (levels l >= 1, read by many neighbouring tiles,
// so mostly L1 hits) with 4-byte cp.async copies, one tile ahead.  The tile's
// own full-resolution row (level 0, streamed from DRAM once) comes
//   without TMA (TMA = false): the same way, one cp.async per thread;
//   with TMA (TMA = true):     as one TMA box per channel (a 1-D tensor map
//                              over the call's latents), which the group's
//                              issuing warp loads into one of two buffers two
//                              tiles ahead, right after the decoders have
//                              handed over the tile that used that buffer.
//                              The issuing warp also waits for the box of the
//                              next tile and then arrives on the group's
//                              col_ready barrier as its 129th participant, so
//                              the decoders, which read level 0 after that
//                              barrier, wait on nothing more than without TMA
//                              (an extra wait per tile in the decoders cost
//                              c5 9-14 %).
#pragma once

#include <cuda_fp16.h>
#include <cuda_fp8.h>

#include <type_traits>

#include "pic_common.cuh"
#include "pic_kernels.h"
#include "tc_ptx.cuh"

namespace pic {
namespace {

using namespace tc;

constexpr int kTile = 128;
constexpr uint32_t kSpinLimit = kWaitPolls;  // a few seconds of polling at most per wait

__host__ __device__ constexpr int round_up(int v, int m) { return (v + m - 1) / m * m; }
__host__ __device__ constexpr int pow2_at_least(int v) {
  int p = 32;
  while (p < v) p *= 2;
  return p;
}

// Byte offset of element (row, k) in a [rows][K] fp16 tile stored K-major in
// the canonical no-swizzle layout: core matrix (row/8, k/8) at
// (row/8) * SBO + (k/8) * LBO with LBO = 128 B and SBO = 16 K bytes.
__host__ __device__ constexpr uint32_t kmaj(int row, int k, int K) {
  return static_cast<uint32_t>((row >> 3) * (K * 16) + (k >> 3) * 128 + (row & 7) * 16 + (k & 7) * 2);
}
// The same for a [rows][K] tile of 8-bit elements: core matrix (row/8, k/16),
// LBO = 128 B, SBO = 8 K bytes.
__host__ __device__ constexpr uint32_t kmaj8(int row, int k, int K) {
  return static_cast<uint32_t>((row >> 3) * (K * 8) + (k >> 4) * 128 + (row & 7) * 16 + (k & 15));
}

// Feature staging per segment of the tile row: a warp's 32 pixels (offset
// 32 (warp & 3) within the tile; single-channel nets) or the group's whole
// 128 (nets with more channels, whose per-warp buffers would take more
// staging registers).  A segment of SEG pixels needs at most NCOL(l) =
// SEG/2^l + 4 source columns of level l >= 1.  Its threads first
// interpolate those columns vertically (rows v0, v1 of the level, weight
// beta) into the segment's small shared buffer -- one item per (level,
// channel, column), spread over them -- and every pixel then interpolates
// horizontally between two buffer entries.  A warp segment needs only a
// __syncwarp between the two passes (the group barrier it replaces measured
// 4-5 % of the c5 time); a group segment waits on the group's col_ready
// mbarrier.  Column indices are clamped into [0, W_l - 1] when the buffer is
// filled, which reproduces the edge clamp of the bilinear definition.
__host__ __device__ constexpr int ncol(int l, int seg) { return (seg >> l) + 4; }
static_assert(kTile == kTcTile, "one tile size for the kernels and the host's TMA boxes");

// One TMA buffer (TMA kernels): a slot per channel for the tile's level-0
// row segment, each holding one box of kTmaRowBox 4-byte words and starting
// on a 128-byte boundary (a tiled TMA copy's shared-memory destination must
// be 128-byte aligned).
template <int C>
struct TmaSlots {
  static constexpr int slot() { return (kTmaRowBox * 4 + 127) / 128 * 128; }
  static constexpr int off(int c) { return c * slot(); }  // bytes
  static constexpr int total() { return C * slot(); }
  static constexpr int boxes() { return C; }
  static constexpr int tx_bytes() { return C * kTmaRowBox * 4; }  // the stage mbarrier's count
};

template <int L, int C, int SEG>
struct ColLayout {
  // float offset of (level l, channel c) inside a segment's column buffer
  static constexpr int off(int l, int c) {
    int o = 0;
    for (int k = 1; k < l; ++k) o += C * ncol(k, SEG);
    return o + c * ncol(l, SEG);
  }
  static constexpr int total() { return off(L, 0); }
};

template <int C_, int NL_, int D0_, int N_, int ACT_, int NWG_, bool LO8_ = false, int NR_ = N_>
struct TcNet {
  static constexpr int C = C_, NL = NL_, D0 = D0_, N = N_, ACT = ACT_, NWG = NWG_;
  static constexpr bool LO8 = LO8_;
  // hidden neurons the net has (N is that rounded up to the MMA's N step):
  // columns NR .. N - 1 hold zero weights and bias, so their accumulators are
  // exactly +0 and the epilogues write +0 there without computing anything
  static constexpr int NR = NR_;
  static_assert(NR_ >= 1 && NR_ <= N_, "real hidden width within the tile");
  static constexpr int SEG = C == 1 ? 32 : kTile;  // staging segment: a warp's pixels or the group's
  static constexpr int NSEG = kTile / SEG;         // segments (column buffers) per group
  // Hidden operand layout in tensor memory: per 16-value chunk the hi and the
  // lo columns adjacent (one 16-column store; single-channel nets, measured
  // 1 % faster on c5), else all hi columns, then all lo columns.
  static constexpr bool ADJ = C == 1 && !LO8;
  static constexpr float kS = LO8 ? 64.0f : 1.0f;  // scale of the hidden activations (LO8)
  static constexpr int L = D0 / C;
  static constexpr int K1 = round_up(2 * D0 + 1, 16);
  // Output layer on the CUDA cores (fp32, one MMA round trip less per tile)
  // when the hidden width is small or the net deep enough that the saved
  // round trip outweighs the extra FMAs; else on the tensor cores (N = 16
  // tile, split operands).  Measured: faster for 8-16-16-16-3 and
  // 16-64-64-64-3, slower for 7-64-64-3.
  static constexpr bool OUTCC = (N <= 32) || (NL >= 4);
  static constexpr int NOUT = 16;
  static constexpr int NISSUE = NWG;                  // one MMA-issuing warp per group
  static constexpr int THREADS = NWG * 128 + 32 * NISSUE;
  static constexpr int MMA_WARP = NWG * 4;            // first issuing warp (also owns TMEM)
  // Registers per thread that still let one CTA fit an SM: the warps are
  // spread over the 4 sub-partitions, each with a 16K-register file.
  static constexpr int WARPS_PER_SMSP = (THREADS / 32 + 3) / 4;
  static constexpr int MAXREG_RAW = 16384 / (32 * WARPS_PER_SMSP) / 8 * 8;
  static constexpr int MAXREG = MAXREG_RAW > 255 ? 255 : MAXREG_RAW;
  // Registers moved at run time (setmaxnreg) from the issuing warpgroup,
  // which needs few, to the decoding warpgroups.  The two budgets together
  // must not exceed what the CTA was launched with (MAXREG per thread; the
  // host refuses a build whose kernel does not use exactly MAXREG), or the
  // increase would wait forever.
  static constexpr int REG_ISSUE = 64;
  static constexpr int REG_DECODE_RAW = (MAXREG * THREADS - REG_ISSUE * 32 * NISSUE) / (NWG * 128) / 8 * 8;
  static constexpr int REG_DECODE = REG_DECODE_RAW > 248 ? 248 : REG_DECODE_RAW;
  static constexpr int CTRL = 256;
  static constexpr int B1_BYTES = N * K1 * 2;
  static constexpr int KB = N + 16;                      // [W | b 0..0]
  static constexpr int BH_BYTES = N * KB * 2;
  // output layer: [W | b 0..0] padded to NOUT rows for the tensor cores; on
  // the CUDA cores fp32, per pair q of inputs 8 floats (w0 w0 | w1 w1 |
  // w2 w2 | 0 0 at inputs 2q, 2q+1), then the 3 biases
  static constexpr int BO_BYTES = OUTCC ? (N / 2) * 32 + 16 : NOUT * KB * 2;
  // LO8: e4m3 copies of the hidden layers' and the output layer's W, K-major
  // [rows][N] bytes (core matrices of 8 rows x 16 bytes)
  static constexpr int BL_BYTES = LO8 ? N * N : 0;
  static constexpr int BLO_BYTES = LO8 ? NOUT * N : 0;
  static constexpr int ONES_BYTES = kTile * 16 * 2;      // constant A tile [1 0..0] per row
  static constexpr int OFF_B1 = CTRL;
  static constexpr int OFF_BH = OFF_B1 + B1_BYTES;
  static constexpr int OFF_BO = OFF_BH + (NL - 2) * BH_BYTES;
  static constexpr int OFF_BL = round_up(OFF_BO + BO_BYTES, 128);
  static constexpr int OFF_BLO = OFF_BL + (NL - 2) * BL_BYTES;
  static constexpr int OFF_ONES = round_up(OFF_BLO + BLO_BYTES, 128);
  static constexpr int OFF_WG = round_up(OFF_ONES + ONES_BYTES, 128);
  static constexpr int A1_BYTES = kTile * K1 * 2;
  static constexpr int COL_BYTES = round_up(NSEG * ColLayout<L, C, SEG>::total() * 4, 128);
  static constexpr int NITEM_PER_THREAD = (ColLayout<L, C, SEG>::total() + SEG - 1) / SEG;
  static constexpr int STAGE_SLOTS = C + 2 * NITEM_PER_THREAD;  // raw int32 loads per thread
  static constexpr int STAGE_BYTES = STAGE_SLOTS * kTile * 4;
  static constexpr int WG_BYTES = A1_BYTES + COL_BYTES + STAGE_BYTES;
  static constexpr int SMEM = OFF_WG + NWG * WG_BYTES;
  // TMA kernels: the per-thread staging slots give way to two TMA buffers
  static constexpr int TBUF_BYTES = round_up(TmaSlots<C>::total(), 128);
  static constexpr int WG_BYTES_TMA = WG_BYTES + 2 * TBUF_BYTES;
  static constexpr int SMEM_TMA = OFF_WG + NWG * WG_BYTES_TMA;
  static constexpr int TMEM_COLS = pow2_at_least(NWG * 2 * N);
  static_assert(N % 16 == 0 && N >= 16 && N <= 128, "hidden width must be 16..128, multiple of 16");
  static_assert(NL >= 2, "the tensor-core path needs at least one hidden layer");
  static_assert(!LO8 || (ACT == ACT_RELU && !OUTCC && N % 32 == 0),
                "the fp8 lo term: ReLU nets, output layer on the tensor cores, K steps of 32");
  static_assert(TMEM_COLS <= 512, "tensor memory holds 512 columns");
  static_assert(NISSUE == 4 && MMA_WARP % 4 == 0, "the issuing warps form one warpgroup");
  static_assert(REG_DECODE >= MAXREG && REG_DECODE * NWG * 128 + REG_ISSUE * 32 * NISSUE <= MAXREG * THREADS,
                "register split within the launch budget");
  static_assert(8 * (6 * NWG + NISSUE) <= 224, "control block holds the barriers");
  static_assert(TmaSlots<C>::boxes() <= 32, "a tile's TMA boxes, one per lane of a warp");
  static_assert(WG_BYTES % 128 == 0 && TBUF_BYTES % 128 == 0 && OFF_WG % 128 == 0,
                "TMA buffers on 128-byte boundaries");
};

// Bounded mbarrier wait: at most `limit` polls (the launch's spin_limit;
// kWaitPolls in production).  Returns false (and raises the abort flag and
// the handle's status word) if the phase does not complete in time, or if
// another thread has already aborted.
__device__ __forceinline__ bool wait_bounded(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                             int* status, uint32_t limit) {
  if (mbar_test_wait(bar, parity)) return true;  // a completed phase: no blocking probe
  for (uint32_t i = 0; i < limit; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 63u) == 63u) {
      if (*abort_flag) return false;
      if (i > 4096) __nanosleep(64);
    }
  }
  *abort_flag = 1;
  atomicOr(status, 1);
  return false;
}

__device__ __forceinline__ __half ldh(const __half* p) {
  return __ushort_as_half(__ldg(reinterpret_cast<const unsigned short*>(p)));
}

// Fills the weight operands and biases of one image into shared memory
// (threads tid = 0 .. nthr-1 of the decoding warpgroups).
template <class Net>
__device__ __forceinline__ void load_weights_tc(uint8_t* smem, const __half* w,
                                                const int (&dims)[Net::NL + 1], int tid, int nthr) {
  constexpr int N = Net::N, D0 = Net::D0, K1 = Net::K1, NL = Net::NL, KB = Net::KB;
  const __half zero = __float2half_rn(0.0f);
  // LO8: S times an fp16 value (exact: S is a power of two and |v| < 1024)
  auto scaled = [](__half v) {
    if constexpr (Net::LO8) return __float2half_rn(__half2float(v) * Net::kS);
    else return v;
  };
  // layer 0: [W | W | b | 0] (LO8: S W, S b)
  {
    const int d1 = dims[1];
    const __half* W0 = w;
    const __half* b0 = w + d1 * D0;
    for (int e = tid; e < N * K1; e += nthr) {
      const int n = e / K1, j = e - n * K1;
      __half v = zero;
      if (n < d1) {
        if (j < D0) v = scaled(ldh(W0 + n * D0 + j));
        else if (j < 2 * D0) v = scaled(ldh(W0 + n * D0 + (j - D0)));
        else if (j == 2 * D0) v = scaled(ldh(b0 + n));
      }
      *reinterpret_cast<__half*>(smem + Net::OFF_B1 + kmaj(n, j, K1)) = v;
    }
  }
  // hidden layers and output: [W | b 0..0] (LO8: S b), zero padded to N (or
  // 16) rows; LO8 also the e4m3 copy of W, [rows][N] bytes
  const __half* p = w + dims[1] * D0 + dims[1];
#pragma unroll
  for (int k = 1; k < NL; ++k) {
    const int din = dims[k], dout = dims[k + 1];
    const bool out_layer = (k == NL - 1);
    if constexpr (Net::OUTCC) {
      if (out_layer) {  // 3 x din, fp16 -> fp32 (exact), in the pair layout of BO_BYTES
        float* wo = reinterpret_cast<float*>(smem + Net::OFF_BO);
        for (int e = tid; e < (N / 2) * 8; e += nthr) {
          const int q = e >> 3, o = (e >> 1) & 3, j = 2 * q + (e & 1);
          wo[e] = (o < 3 && j < din) ? __half2float(ldh(p + o * din + j)) : 0.0f;
        }
        if (tid < 4) wo[4 * N + tid] = tid < 3 ? __half2float(ldh(p + 3 * din + tid)) : 0.0f;
        break;
      }
    }
    const int rows = out_layer ? Net::NOUT : N;
    uint8_t* base = smem + (out_layer ? Net::OFF_BO : Net::OFF_BH + (k - 1) * Net::BH_BYTES);
    const __half* Wk = p;
    const __half* bk = p + dout * din;
    for (int e = tid; e < rows * KB; e += nthr) {
      const int n = e / KB, j = e - n * KB;
      __half v = zero;
      if (n < dout) {
        if (j < din) v = ldh(Wk + n * din + j);
        else if (j == N) v = scaled(ldh(bk + n));
      }
      *reinterpret_cast<__half*>(base + kmaj(n, j, KB)) = v;
    }
    if constexpr (Net::LO8) {
      uint8_t* lo = smem + (out_layer ? Net::OFF_BLO : Net::OFF_BL + (k - 1) * Net::BL_BYTES);
      for (int e = tid; e < rows * N; e += nthr) {
        const int n = e / N, j = e - n * N;
        uint8_t v = 0;
        if (n < dout && j < din)
          v = __nv_cvt_float_to_fp8(__half2float(ldh(Wk + n * din + j)), __NV_SATFINITE, __NV_E4M3);
        lo[kmaj8(n, j, N)] = v;
      }
    }
    p = bk + dout;
  }
}

// Splits v into (hi, lo) fp32 parts: hi = v rounded toward zero to fp16
// (exactly representable), lo = v - hi (exact in fp32).
__device__ __forceinline__ void split_hi_lo(float v, float& hi, float& lo) {
  hi = __half2float(__float2half_rz(v));
  lo = v - hi;
}

// The last hidden layer's epilogue fused with the output layer on the CUDA
// cores (Net::OUTCC): activation, then rgb = W_out h + b_out in fp32 (packed
// FMAs on pairs of hidden values; the weights are the fp16 values held
// exactly in fp32, layout of Net::BO_BYTES).
template <class Net>
__device__ __forceinline__ void output_layer_cc(const uint8_t* smem, uint32_t t_acc, float (&rgb)[3]) {
  constexpr int N = Net::N;
  const float* wo = reinterpret_cast<const float*>(smem + Net::OFF_BO);
  unsigned long long s0 = 0ull, s1 = 0ull, s2 = 0ull;  // (+0, +0) pairs
#pragma unroll
  for (int h0 = 0; h0 < N; h0 += 16) {
    uint32_t acc[16];
    tmem_ld16(t_acc + h0, acc);
    tmem_ld_wait();
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      if (h0 + 2 * q >= Net::NR) continue;  // padding: act(+0) = +0 adds nothing
      unsigned long long hv;
      if constexpr (Net::ACT == ACT_GELU) {
        hv = gelu_approx2(pack2(__uint_as_float(acc[2 * q]), __uint_as_float(acc[2 * q + 1])));
      } else {
        hv = pack2(fmaxf(__uint_as_float(acc[2 * q]), 0.0f),
                   fmaxf(__uint_as_float(acc[2 * q + 1]), 0.0f));
      }
      const float4 wa = *reinterpret_cast<const float4*>(wo + 8 * (h0 / 2 + q));
      const float4 wb = *reinterpret_cast<const float4*>(wo + 8 * (h0 / 2 + q) + 4);
      s0 = fma2(pack2(wa.x, wa.y), hv, s0);
      s1 = fma2(pack2(wa.z, wa.w), hv, s1);
      s2 = fma2(pack2(wb.x, wb.y), hv, s2);
    }
  }
  const float2 r0 = unpack2(s0), r1 = unpack2(s1), r2 = unpack2(s2);
  rgb[0] = r0.x + r0.y + wo[4 * N + 0];
  rgb[1] = r1.x + r1.y + wo[4 * N + 1];
  rgb[2] = r2.x + r2.y + wo[4 * N + 2];
}

// Hidden epilogue of one pixel (TMEM lane): accumulator -> activation ->
// hi/lo split -> the next layer's A operand in TMEM, 16 values at a time
// (fewer live registers): chunk c's hi pairs at t_a + 16c and lo pairs at
// t_a + 16c + 8 (Net::ADJ), else hi pairs at t_a + 8c, lo at t_a + N/2 + 8c.
template <class Net>
__device__ __forceinline__ void hidden_epilogue(uint32_t t_acc, uint32_t t_a) {
  constexpr int N = Net::N;
#pragma unroll
  for (int h0 = 0; h0 < N; h0 += 16) {
    uint32_t acc[16];
    tmem_ld16(t_acc + h0, acc);
    tmem_ld_wait();
    uint32_t hl[16];  // [0, 8): hi pairs, [8, 16): lo pairs
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      if (h0 + 2 * q >= Net::NR) {  // padding columns: act(+0) = +0, split into +0 and +0
        hl[q] = 0u;
        hl[8 + q] = 0u;
        continue;
      }
      float a = __uint_as_float(acc[2 * q]);
      float bb = __uint_as_float(acc[2 * q + 1]);
      if constexpr (Net::ACT == ACT_GELU) {
        const float2 g = unpack2(gelu_approx2(pack2(a, bb)));
        a = g.x;
        bb = g.y;
      }
      // hi = fp16 truncation (ReLU folded in), lo = fp16 of v - hi (one mixed FMA)
      split_pair<Net::ACT != ACT_GELU>(a, bb, hl[q], hl[8 + q]);
    }
    if constexpr (Net::ADJ) {
      tmem_st16(t_a + h0, hl);
    } else {
      tmem_st8(t_a + h0 / 2, hl);
      tmem_st8(t_a + N / 2 + h0 / 2, hl + 8);
    }
  }
  tmem_st_wait();
}

// LO8: hidden epilogue with the lo terms in e4m3: hi pairs at t_a (N/2
// columns), lo quads at t_a + N/2 (N/4 columns), 16 values at a time.
template <class Net>
__device__ __forceinline__ void hidden_epilogue_lo8(uint32_t t_acc, uint32_t t_a) {
  constexpr int N = Net::N;
#pragma unroll
  for (int h0 = 0; h0 < N; h0 += 16) {
    uint32_t acc[16];
    tmem_ld16(t_acc + h0, acc);
    tmem_ld_wait();
    uint32_t hi[8], lo[4];
#pragma unroll
    for (int q = 0; q < 8; q += 2) {
      uint16_t l0, l1;
      split_pair_e4m3(__uint_as_float(acc[2 * q]), __uint_as_float(acc[2 * q + 1]), hi[q], l0);
      split_pair_e4m3(__uint_as_float(acc[2 * q + 2]), __uint_as_float(acc[2 * q + 3]), hi[q + 1], l1);
      lo[q / 2] = static_cast<uint32_t>(l0) | (static_cast<uint32_t>(l1) << 16);
    }
    tmem_st8(t_a + h0 / 2, hi);
    tmem_st4(t_a + N / 2 + h0 / 4, lo);
  }
  tmem_st_wait();
}

// The tile cursor (row yy, tile column xx) advanced by NWG tiles.
template <int NWG>
__device__ __forceinline__ void advance_tile(int& yy, int& xx, int tpr) {
  xx += NWG;
  while (xx >= tpr) {
    xx -= tpr;
    ++yy;
  }
}

template <class Net, bool FL, bool TMA>
__global__ void __launch_bounds__(Net::THREADS) __maxnreg__(Net::MAXREG)
    tc_decode_kernel(const DecodeParams p, const __grid_constant__ TmaParams tp) {
  constexpr int N = Net::N, NL = Net::NL, C = Net::C, L = Net::L, D0 = Net::D0, NWG = Net::NWG;
  constexpr int K1 = Net::K1;
  constexpr int WGB = TMA ? Net::WG_BYTES_TMA : Net::WG_BYTES;
  using TS = TmaSlots<C>;
  constexpr int SEG = Net::SEG;
  using CL = ColLayout<L, C, SEG>;
  constexpr int NITEM = CL::total();  // column items of one segment
  constexpr int J = (NITEM + SEG - 1) / SEG;  // column items per thread (0 if L == 1)
  constexpr int JJ = J > 0 ? J : 1;
  extern __shared__ __align__(1024) uint8_t smem[];

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t sbase = smem_addr(smem);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + 224);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + 232);
  // mbarriers, 8 bytes each: per group w a1_full (features written),
  // a_full (hidden operand written), acc_full (MMAs done), col_ready; one drain.
  const uint32_t bar_a1 = sbase;
  const uint32_t bar_a = sbase + 8 * NWG;
  const uint32_t bar_c = sbase + 16 * NWG;
  const uint32_t bar_col = sbase + 24 * NWG;
  const uint32_t bar_drain = sbase + 32 * NWG;  // + 8 m for issuing warp m
  // TMA kernels: per group two stage_full barriers (its boxes for the tile
  // using buffer 0 / 1 have landed), at bar_stage + 16 w + 8 buffer
  const uint32_t bar_stage = bar_drain + 8 * Net::NISSUE;

  if (threadIdx.x == 0) {
    for (int w = 0; w < NWG; ++w) {
      mbar_init(bar_a1 + 8 * w, 128);
      mbar_init(bar_a + 8 * w, 128);
      mbar_init(bar_c + 8 * w, 1);
      mbar_init(bar_col + 8 * w, TMA ? 129 : 128);  // TMA: + the issuing warp's arrival
    }
    for (int m = 0; m < Net::NISSUE; ++m) mbar_init(bar_drain + 8 * m, 1);
    if constexpr (TMA)
      for (int q = 0; q < 2 * NWG; ++q) mbar_init(bar_stage + 8 * q, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == Net::MMA_WARP) {
    tmem_alloc(smem_addr(tmem_slot), Net::TMEM_COLS);
    tmem_relinquish();
  }
  for (int e = threadIdx.x; e < kTile * 2; e += blockDim.x) {  // 16-byte chunks of the ones tile
    const int row = e >> 1, kc = e & 1;
    sts128(sbase + Net::OFF_ONES + kmaj(row, kc * 8, 16), kc == 0 ? 0x00003C00u : 0u, 0u, 0u, 0u);
  }
  fence_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  const long long chunk = (p.total_tiles + gridDim.x - 1) / gridDim.x;
  const long long t_begin = blockIdx.x * chunk;
  const long long t_end = min(t_begin + chunk, p.total_tiles);
  const __half* wts = static_cast<const __half*>(p.weights);
  const long long plane = static_cast<long long>(p.H) * p.W;
  // x-taps repeat from tile to tile when every level's width is exactly W / 2^l
  // (and 2^l divides the 128-pixel tile origin, i.e. l <= 7)
  const bool fast_x = (L - 1 <= 7) && (p.W % (1 << (L - 1))) == 0;

  uint32_t acc_phase = 0;  // warpgroup threads: parity of their acc_full
  uint32_t col_phase = 0;  // warpgroup threads: parity of their col_ready
  uint32_t a1_phase = 0;   // MMA warp: bit w = parity of a1_full[w]
  uint32_t a_phase = 0;    // MMA warp: bit w = parity of a_full[w]
  uint32_t stage_phase = 0;  // TMA, issuing warps: bit q = parity of the next box set issued on q
  uint32_t stage_wait = 0;   // TMA, issuing warps: bit q = parity of the next box set to wait for on q

  // Each role runs its own loop over the images of its tile range, so that
  // it can hold its own register budget: the issuing warpgroup gives
  // registers back, the decoding warpgroups take them (setmaxnreg).
  if (warp < 4 * NWG) {
    setmaxnreg_inc<Net::REG_DECODE>();
    for (long long seg = t_begin; seg < t_end;) {
      const int b = static_cast<int>(seg / p.tiles_per_image);
      const long long seg_end = min(t_end, static_cast<long long>(b + 1) * p.tiles_per_image);
      __syncthreads();  // all MMAs and reads of the previous image's weights are done
      {
        int dims[NL + 1];
#pragma unroll
        for (int k = 0; k <= NL; ++k) dims[k] = p.dims[k];
        load_weights_tc<Net>(smem, wts + b * p.params_per_image, dims, threadIdx.x, 4 * NWG * 32);
      }
      fence_async_smem();
      __syncthreads();
      const int n_tiles = static_cast<int>(seg_end - seg);
      const long long tile0 = seg - static_cast<long long>(b) * p.tiles_per_image;  // in-image index
      {
        // ------------------------------------------------------------ warpgroup
        const int w = warp >> 2;
        const int r = ((warp & 3) << 5) | lane;  // tile row = TMEM lane = pixel
        uint8_t* a1 = smem + Net::OFF_WG + w * WGB;
        const uint32_t a1_s = smem_addr(a1);
        // this thread's segment: its column buffer, its offset xo in the tile
        // row, and the thread's place sr in it
        const int sid = SEG == kTile ? 0 : (warp & 3);
        float* colbuf = reinterpret_cast<float*>(a1 + Net::A1_BYTES) + sid * NITEM;
        const int xo = sid * SEG;
        const int sr = r - xo;
        const uint32_t lane_off = static_cast<uint32_t>((warp & 3) * 32) << 16;
        const uint32_t t_acc = tmem + lane_off + static_cast<uint32_t>(w * 2 * N);
        const uint32_t t_a = t_acc + N;  // hi in [0, N/2), lo in [N/2, N)
        const uint32_t my_a1 = bar_a1 + 8 * w, my_a = bar_a + 8 * w, my_c = bar_c + 8 * w,
                       my_col = bar_col + 8 * w;
        const int32_t* lat = p.latents + b * p.lat_per_image;
        float step[L];
#pragma unroll
        for (int l = 0; l < L; ++l) step[l] = FL ? 1.0f : __ldg(p.steps + b * L + l);

        // This thread's column items: level, column, and the level's geometry.
        int it_l[JJ], it_i[JJ], it_W[JJ], it_H[JJ];
        long long it_off[JJ];
        float it_sy[JJ], it_sx[JJ];
        float it_beta[JJ];  // vertical weight of each item for the tile last prefetched
#pragma unroll
        for (int j = 0; j < J; ++j) {
          int e = sr + SEG * j, l = 0, c = 0, i = 0;
          if (e < NITEM) {
#pragma unroll
            for (int lv = 1; lv < L; ++lv)
#pragma unroll
              for (int cc = 0; cc < C; ++cc)
                if (e >= CL::off(lv, cc) && e < CL::off(lv, cc) + ncol(lv, SEG)) {
                  l = lv;
                  c = cc;
                  i = e - CL::off(lv, cc);
                }
          }
          it_l[j] = l;  // l == 0 marks an idle slot
          it_i[j] = i;
          const LevelGeom lg = p.lv[l];
          it_W[j] = lg.W;
          it_H[j] = lg.H;
          it_off[j] = lg.off + static_cast<long long>(c) * lg.H * lg.W;
          it_sy[j] = lg.sy;
          it_sx[j] = lg.sx;
        }
        // Relative x-taps of pixel r for each level (used when fast_x): the
        // source coordinate of pixel x0 + r, relative to column (x0 + xo)/2^l
        // - 1, is ((xo mod 2^l) + lane + 1/2) / 2^l - 1/2 + 1 (x0 is a
        // multiple of 128 >= 2^l, so this does not depend on the tile).
        int rel[L];
        float fx[L];
#pragma unroll
        for (int l = 1; l < L; ++l) {
          const int off = (xo & ((1 << l) - 1)) + sr;
          const float sx = (static_cast<float>(off) + 0.5f) * (1.0f / static_cast<float>(1 << l)) - 0.5f;
          const float fl = floorf(sx);
          rel[l] = static_cast<int>(fl) + 1;
          fx[l] = sx - fl;
        }

        // Global loads tile (y, x0) needs -- the level-0 values of pixel r and
        // the raw texel pairs of this thread's column items -- issued as
        // asynchronous copies into this thread's column of the staging buffer
        // (slot s of thread r at stage[s * 128 + r]); nothing waits on them
        // until the features are computed.
        const uint32_t stage_s = a1_s + Net::A1_BYTES + Net::COL_BYTES;
        const int* stage = reinterpret_cast<const int*>(a1 + Net::A1_BYTES + Net::COL_BYTES);
        auto prefetch = [&](int y, int x0) {
          if constexpr (!TMA) {  // else the level-0 row arrives as the issuing warp's TMA boxes
            const int xc = min(x0 + r, p.W - 1);
#pragma unroll
            for (int c = 0; c < C; ++c)
              cp_async4(stage_s + (c * kTile + r) * 4, lat + c * plane + static_cast<long long>(y) * p.W + xc);
          }
#pragma unroll
          for (int j = 0; j < J; ++j) {
            const int l = it_l[j];
            if (l > 0) {
              const Tap ty = bilinear_tap(y, it_sy[j], it_H[j]);
              it_beta[j] = ty.frac;
              const int u_start =
                  fast_x ? ((x0 + xo) >> l) - 1 : bilinear_tap(x0 + xo, it_sx[j], it_W[j]).i0;
              const int u = min(max(u_start + it_i[j], 0), it_W[j] - 1);
              const int32_t* pl = lat + it_off[j] + u;
              cp_async4(stage_s + ((C + 2 * j) * kTile + r) * 4, pl + ty.i0 * it_W[j]);
              cp_async4(stage_s + ((C + 2 * j + 1) * kTile + r) * 4, pl + ty.i1 * it_W[j]);
            }
          }
          cp_async_commit();
        };

        // TMA kernels: the level-0 row of the group's k-th tile sits in TMA
        // buffer k & 1 once the tile's col_ready phase has completed (the
        // issuing warp arrives there only after the box has landed), channel
        // c's box from latent word s_c & ~3 on, where
        // s_c is the word of (c, y, x0) in the call's latent buffer; pixel r
        // is box word (s_c & 3) + r.  Only the low two bits of the word index
        // are used, so 32-bit wrap-around is harmless.
        const uint8_t* tbuf = a1 + Net::A1_BYTES + Net::COL_BYTES + Net::STAGE_BYTES;
        const unsigned img_word =
            static_cast<unsigned>(b) * static_cast<unsigned>(p.lat_per_image);

        // Features of the group's k-th tile (y, x0) from its staged loads ->
        // A1 (shared).  Returns false if a wait gave up.
        auto features = [&](int y, int x0, int k) -> bool {
          cp_async_wait_all();  // this thread's staged loads have landed
          // vertical pass into the column buffer
#pragma unroll
          for (int j = 0; j < J; ++j) {
            const int l = it_l[j];
            if (l > 0) {
              const float beta = it_beta[j];  // set by the prefetch of this tile
              const int t0 = stage[(C + 2 * j) * kTile + r], t1 = stage[(C + 2 * j + 1) * kTile + r];
              colbuf[sr + SEG * j] = step[l] * lat_lerp<FL>(t0, t1, beta);
            }
          }
          if constexpr (TMA || SEG == kTile) {
            // the group's barrier: the group's column buffer is complete, and
            // (TMA) the issuing warp hands over the tile's level-0 boxes there
            // (its 129th arrival)
            mbar_arrive(my_col);
            if (!__all_sync(0xffffffffu, wait_bounded(my_col, col_phase, abort_flag, p.status, p.spin_limit)))
              return false;
            col_phase ^= 1u;
          } else {
            __syncwarp();  // this warp's column buffer is complete
          }
          // horizontal pass + level 0
          const int xc = min(x0 + r, p.W - 1);
          float f[D0];
#pragma unroll
          for (int c = 0; c < C; ++c) {
            if constexpr (TMA) {
              const unsigned sc = img_word + static_cast<unsigned>(c * plane + y * p.W + x0);
              const int* slot = reinterpret_cast<const int*>(tbuf + (k & 1) * Net::TBUF_BYTES + TS::off(c));
              f[c] = step[0] * lat_value<FL>(slot[(sc & 3u) + r]);
            } else {
              f[c] = step[0] * lat_value<FL>(stage[c * kTile + r]);
            }
          }
#pragma unroll
          for (int l = 1; l < L; ++l) {
            int i0, i1;
            float a;
            if (fast_x) {
              i0 = rel[l];
              i1 = rel[l] + 1;
              a = fx[l];
            } else {
              const LevelGeom lg = p.lv[l];
              const int u_start = bilinear_tap(x0 + xo, lg.sx, lg.W).i0;
              const Tap tx = bilinear_tap(xc, lg.sx, lg.W);
              i0 = min(max(tx.i0 - u_start, 0), ncol(l, SEG) - 1);
              i1 = min(max(tx.i1 - u_start, 0), ncol(l, SEG) - 1);
              a = tx.frac;
            }
#pragma unroll
            for (int c = 0; c < C; ++c) {
              const float* cb = colbuf + CL::off(l, c);
              const float v0 = cb[i0], v1 = cb[i1];
              f[l * C + c] = fmaf(a, v1 - v0, v0);
            }
          }
          // hi/lo split, the constant-1 bias column, padding -> A1
          float v[K1];
#pragma unroll
          for (int j = 0; j < K1; ++j) v[j] = 0.0f;
#pragma unroll
          for (int j = 0; j < D0; ++j) split_hi_lo(f[j], v[j], v[D0 + j]);
          v[2 * D0] = 1.0f;
#pragma unroll
          for (int kc = 0; kc < K1 / 8; ++kc)
            sts128(a1_s + kmaj(r, kc * 8, K1), pack_f16x2(v[kc * 8 + 0], v[kc * 8 + 1]),
                   pack_f16x2(v[kc * 8 + 2], v[kc * 8 + 3]), pack_f16x2(v[kc * 8 + 4], v[kc * 8 + 5]),
                   pack_f16x2(v[kc * 8 + 6], v[kc * 8 + 7]));
          fence_async_smem();
          return true;
        };

        // Tile cursor (row y, tile column tx) of this group's current tile and
        // of the one after it, advanced by NWG tiles without divisions.
        const int tpr = p.tiles_per_row;
        int cy = static_cast<int>((tile0 + w) / tpr);
        int ctx = static_cast<int>((tile0 + w) - static_cast<long long>(cy) * tpr);

        bool ok = true;
        if (w < n_tiles) {
          prefetch(cy, ctx * kTile);
          ok = features(cy, ctx * kTile, 0);
          // p.test_fault (tests of the bounded waits only; 0 in every
          // production launch): one thread of CTA 0's first group withholds
          // its first a1_full arrival, so the issuing warp's wait runs out
          const bool withhold = p.test_fault && blockIdx.x == 0 && w == 0 && r == 5 && seg == t_begin;
          if (ok && !withhold) mbar_arrive(my_a1);
        }
        for (int i = w; i < n_tiles && ok; i += NWG) {
          if (__any_sync(0xffffffffu, *abort_flag != 0)) break;
          const int y = cy;
          const int x0 = ctx * kTile;
          int ny = cy, ntx = ctx;
          advance_tile<NWG>(ny, ntx, tpr);
          const bool has_next = i + NWG < n_tiles;
          const int knext = (i - w) / NWG + 1;  // the group's index of the next tile
          if (has_next) prefetch(ny, ntx * kTile);  // in flight during the first epilogue

          if constexpr (Net::OUTCC) {
            // hidden epilogues up to the last one, which runs the output layer
            for (int k = 0; k < NL - 2 && ok; ++k) {
              if (!__all_sync(0xffffffffu, wait_bounded(my_c, acc_phase, abort_flag, p.status, p.spin_limit))) {
                ok = false;
                break;
              }
              acc_phase ^= 1u;
              tc_fence_after();
              hidden_epilogue<Net>(t_acc, t_a);
              tc_fence_before();
              mbar_arrive(my_a);
              if (k == 0 && has_next) ok = features(ny, ntx * kTile, knext);  // overlaps layer 1
            }
            if (!ok) break;
            if (!__all_sync(0xffffffffu, wait_bounded(my_c, acc_phase, abort_flag, p.status, p.spin_limit))) break;
            acc_phase ^= 1u;
            tc_fence_after();
            float rgb[3];
            output_layer_cc<Net>(smem, t_acc, rgb);
            tc_fence_before();
            if (NL == 2 && has_next) ok = features(ny, ntx * kTile, knext);  // no hidden layer to overlap
            if (has_next && ok) mbar_arrive(my_a1);  // accumulator read: the next tile's layer 0 may start
            const int x = x0 + r;
            if (x < p.W) store_rgb(p, b, y, x, rgb[0], rgb[1], rgb[2]);
            cy = ny;
            ctx = ntx;
            if (!ok) break;
          } else {
            for (int k = 0; k < NL - 1 && ok; ++k) {
              if (!__all_sync(0xffffffffu, wait_bounded(my_c, acc_phase, abort_flag, p.status, p.spin_limit))) {
                ok = false;
                break;
              }
              acc_phase ^= 1u;
              tc_fence_after();
              if constexpr (Net::LO8) hidden_epilogue_lo8<Net>(t_acc, t_a);
              else hidden_epilogue<Net>(t_acc, t_a);
              tc_fence_before();
              mbar_arrive(my_a);
              if (k == 0 && has_next) ok = features(ny, ntx * kTile, knext);  // overlaps layer 1
            }
            if (!ok) break;

            // ---- output layer: bias, clamp, store (LO8: the accumulator holds S o) ----
            if (!__all_sync(0xffffffffu, wait_bounded(my_c, acc_phase, abort_flag, p.status, p.spin_limit))) break;
            acc_phase ^= 1u;
            tc_fence_after();
            uint32_t o[4];
            tmem_ld4(t_acc, o);
            tmem_ld_wait();
            tc_fence_before();
            if (has_next) mbar_arrive(my_a1);  // accumulator read: the next tile's layer 0 may start
            const int x = x0 + r;
            constexpr float inv_s = 1.0f / Net::kS;  // exact: a power of two
            if (x < p.W)
              store_rgb(p, b, y, x, __uint_as_float(o[0]) * inv_s, __uint_as_float(o[1]) * inv_s,
                        __uint_as_float(o[2]) * inv_s);
            cy = ny;
            ctx = ntx;
          }
        }
      }
      seg = seg_end;
    }
    // A wait that gave up may leave this thread's next-tile copies in
    // flight: they land before the CTA's shared memory is released.
    cp_async_wait_all();
  } else {
    setmaxnreg_dec<Net::REG_ISSUE>();
    for (long long seg = t_begin; seg < t_end;) {
      const int b = static_cast<int>(seg / p.tiles_per_image);
      const long long seg_end = min(t_end, static_cast<long long>(b + 1) * p.tiles_per_image);
      __syncthreads();  // all MMAs of the previous image are complete
      __syncthreads();  // the decoding warps have loaded this image's weights
      const int n_tiles = static_cast<int>(seg_end - seg);
      {
        // --------------------------------------------------------------- MMA issuer
        // Warp MMA_WARP + w issues every MMA of group w, in the group's order
        // (its tiles in turn, layers in turn), polling the group's mbarriers
        // in between.  The whole warp runs the control flow (descriptors stay
        // warp-uniform); one elected lane issues the MMAs and the commit.
        // Descriptors depend on the start address only through their low
        // field: base + (offset >> 4).
        const int w = warp - Net::MMA_WARP;
        constexpr uint32_t id_hidden = idesc_f16(128, N);
        constexpr uint32_t id_out = idesc_f16(128, Net::NOUT);
        const uint64_t dA1 = smem_desc(sbase + Net::OFF_WG + w * WGB, 128, 16 * K1);
        const uint64_t dB1 = smem_desc(sbase + Net::OFF_B1, 128, 16 * K1);
        const uint64_t dBH = smem_desc(sbase + Net::OFF_BH, 128, 16 * Net::KB);
        const uint64_t dBO = smem_desc(sbase + Net::OFF_BO, 128, 16 * Net::KB);
        const uint64_t dONES = smem_desc(sbase + Net::OFF_ONES, 128, 16 * 16);
        constexpr uint64_t kStep = 256 >> 4;              // one K-step (16 fp16) = 256 B
        constexpr uint64_t kLayer = Net::BH_BYTES >> 4;   // next hidden layer's weights
        // LO8: the e4m3 copies, K-major with N bytes per row (one K step of
        // 32 e4m3 = two core matrices = 256 B, as for fp16)
        const uint64_t dBL = smem_desc(sbase + Net::OFF_BL, 128, 8 * N);
        const uint64_t dBLO = smem_desc(sbase + Net::OFF_BLO, 128, 8 * N);
        constexpr uint64_t kLayerL = (Net::BL_BYTES >> 4);
        static_assert(Net::WG_BYTES % 16 == 0 && Net::BH_BYTES % 16 == 0, "16-byte aligned operands");
        const uint32_t d = tmem + static_cast<uint32_t>(w * 2 * N);
        const uint32_t ta = d + N;
        const uint32_t my_a1 = bar_a1 + 8 * w, my_a = bar_a + 8 * w, my_c = bar_c + 8 * w;
        // TMA kernels: the level-0 boxes of the group's tile i (of this
        // segment) into buffer buf, one lane per channel; lane 0 first
        // announces the buffer's byte count on its stage_full barrier.
        auto issue_boxes = [&](int y, int x0, int buf) {
          const uint32_t bar = bar_stage + 16 * w + 8 * buf;
          const uint32_t dst = sbase + Net::OFF_WG + w * WGB + Net::WG_BYTES + buf * Net::TBUF_BYTES;
          if (lane == 0) mbar_arrive_expect_tx(bar, TS::tx_bytes());
          __syncwarp();
          if (lane < C) {
            // word indices fit in 32 bits: the host encodes the maps only for
            // buffers of fewer than 2^31 words
            const int start = b * static_cast<int>(p.lat_per_image) + lane * static_cast<int>(plane) +
                              y * p.W + x0;
            // Checked before the copy (never expected to fail: the slot
            // layout and the host's 2^31-word limit rule it out): a
            // misaligned destination or a negative start raises status bit 2
            // and skips the copy, so the decoders' bounded wait reports it.
            const uint32_t d_box = dst + TS::off(lane);
            if ((d_box & 127u) == 0u && start >= 0) tma_load_1d(d_box, &tp.lat, start & ~3, bar);
            else atomicOr(p.status, 2);
          }
          stage_phase ^= 1u << buf;  // parity of the next set on this buffer
        };
        // TMA kernels: waits (bounded) for the boxes of the group's tile in
        // buffer buf, then arrives on the group's col_ready barrier for that
        // tile.  Returns false if the wait gave up.
        auto hand_over = [&](int buf) -> bool {
          const uint32_t bar = bar_stage + 16 * w + 8 * buf;
          const bool landed =
              __all_sync(0xffffffffu, wait_bounded(bar, (stage_wait >> buf) & 1u, abort_flag, p.status, p.spin_limit));
          if (!landed) return false;  // still in flight: the exit drain waits for it
          stage_wait ^= 1u << buf;
          if (lane == 0) mbar_arrive(bar_col + 8 * w);
          return true;
        };
        // Cursor (row, tile column) of the next tile whose boxes this warp
        // issues, advanced by NWG tiles without divisions (as the decoders').
        int by = 0, btx = 0;
        bool ok = true;
        if constexpr (TMA) {
          const long long tile0 = seg - static_cast<long long>(b) * p.tiles_per_image;
          by = static_cast<int>((tile0 + w) / p.tiles_per_row);
          btx = static_cast<int>((tile0 + w) - static_cast<long long>(by) * p.tiles_per_row);
          if (w < n_tiles) issue_boxes(by, btx * kTile, 0);
          advance_tile<NWG>(by, btx, p.tiles_per_row);
          if (w + NWG < n_tiles) issue_boxes(by, btx * kTile, 1);
          advance_tile<NWG>(by, btx, p.tiles_per_row);
          if (w < n_tiles) ok = hand_over(0);  // the first tile's features
        }
        for (int i = w; i < n_tiles && ok; i += NWG) {
          for (int k = 0; k < (Net::OUTCC ? NL - 1 : NL); ++k) {  // OUTCC: no output-layer MMA
            const uint32_t bar = k == 0 ? my_a1 : my_a;
            const uint32_t par = k == 0 ? (a1_phase & 1u) : (a_phase & 1u);
            if (!__all_sync(0xffffffffu, wait_bounded(bar, par, abort_flag, p.status, p.spin_limit))) {
              ok = false;
              break;
            }
            if (k == 0) a1_phase ^= 1u;
            else a_phase ^= 1u;
            if (elect_one()) {
              tc_fence_after();
              if (k == 0) {
#pragma unroll
                for (int s = 0; s < K1 / 16; ++s) mma_f16(d, dA1 + s * kStep, dB1 + s * kStep, id_hidden, s > 0);
              } else {
                const bool out_layer = (k == NL - 1);
                const uint64_t db = out_layer ? dBO : dBH + (k - 1) * kLayer;
                const uint32_t id = out_layer ? id_out : id_hidden;
#pragma unroll
                for (int s = 0; s < N / 16; ++s)  // hi
                  mma_f16_ta(d, ta + (Net::ADJ ? 16 * s : 8 * s), db + s * kStep, id, s > 0);
                if constexpr (Net::LO8) {  // lo in e4m3: K = 32 per MMA, 8 columns of A each
                  const uint64_t dl = out_layer ? dBLO : dBL + (k - 1) * kLayerL;
#pragma unroll
                  for (int s = 0; s < N / 32; ++s) mma_e4m3_ta(d, ta + N / 2 + 8 * s, dl + s * kStep, id, 1);
                } else {
#pragma unroll
                  for (int s = 0; s < N / 16; ++s)  // lo
                    mma_f16_ta(d, ta + (Net::ADJ ? 16 * s + 8 : N / 2 + 8 * s), db + s * kStep, id, 1);
                }
                mma_f16(d, dONES, db + (N / 16) * kStep, id, 1);  // bias: [1 0..0] x [b 0..0]
              }
              mma_commit(my_c);
            }
            __syncwarp();
            if constexpr (TMA) {
              if (k == 0) {
                // The decoders have handed over this tile (its layer-0
                // operand was written before a1_full), so the buffer it used
                // takes the tile two ahead; and the next tile's boxes, issued
                // a tile ago, are handed to the decoders' col_ready barrier.
                const int kk = (i - w) / NWG;
                if (i + 2 * NWG < n_tiles) {
                  issue_boxes(by, btx * kTile, kk & 1);
                  advance_tile<NWG>(by, btx, p.tiles_per_row);
                }
                if (i + NWG < n_tiles && !hand_over((kk + 1) & 1)) {
                  ok = false;
                  break;
                }
              }
            }
          }
        }
      }
      __syncwarp();
      seg = seg_end;
    }
    if constexpr (TMA) {
      // Box sets still in flight (issued, never waited for: a wait gave up
      // first) land before the CTA's shared memory is released: wait for
      // each, bounded.
#pragma unroll
      for (int q = 0; q < 2; ++q)
        if (((stage_phase ^ stage_wait) >> q) & 1u) {
          const uint32_t bar = bar_stage + 16 * (warp - Net::MMA_WARP) + 8 * q;
          for (uint32_t it = 0; it < kSpinLimit; ++it)
            if (mbar_try_wait(bar, (stage_wait >> q) & 1u)) break;
        }
    }
    if (elect_one()) {
      // Every MMA this thread issued must be complete before the memory goes.
      const uint32_t drain = bar_drain + 8 * (warp - Net::MMA_WARP);
      mma_commit(drain);
      int dummy = 0;
      wait_bounded(drain, 0, reinterpret_cast<volatile int*>(&dummy), p.status, kSpinLimit);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == Net::MMA_WARP) {
    tc_fence_after();
    tmem_dealloc(tmem, Net::TMEM_COLS);
  }
}

template <int C, int NL, int D0, int N, int ACT, int NWG, bool FL, bool TMA = false, bool LO8 = false,
          int NR = N>
KernelInfo make_tc(const char* name, const int* dims) {
  using Net = TcNet<C, NL, D0, N, ACT, NWG, LO8, NR>;
  KernelInfo k{};
  k.name = name;
  k.precision = LO8 ? 2 : 1;
  k.latent_format = FL ? 1 : 0;
  k.C = C;
  k.n_layers = NL;
  for (int i = 0; i <= NL; ++i) k.dims[i] = dims[i];
  k.act = ACT;
  k.threads = Net::THREADS;
  k.regs_at_launch = Net::MAXREG;
  k.tile_px = kTile;
  k.smem_bytes = TMA ? Net::SMEM_TMA : Net::SMEM;
  k.tma = TMA ? 1 : 0;
  k.fn = reinterpret_cast<const void*>(&tc_decode_kernel<Net, FL, TMA>);
  return k;
}

}  // namespace
}  // namespace pic
