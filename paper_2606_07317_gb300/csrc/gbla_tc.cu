// Tensor-core (tcgen05 + TMEM + TMA) kernels of the GBLA core for bf16 inputs,
// D in {64, 128}.  Three kernels, launched back to back on one stream:
//
//  tc_state_kernel   (Sec. 2.1 item 1 and item 2, k/v side)
//      Persistent; one CTA per SM.  The 64-token stages of all
//      (batch, group of 128/D heads) sequences are cut into balanced ranges of
//      consecutive stages (ranges may span sequences), so work is even whatever
//      the lengths.  Per range: a pre-pass over its gate logits gives the
//      maximum m over each segment (its part in one sequence); warp 17 streams
//      k tiles (64 tokens + 3 rows of conv history) into a k ring, warp 18 the
//      v tiles into the operand ring; sixteen converter warps run the causal
//      Conv1D of k, phi and the gate weight 2^a' (a' = (a - m) log2 e) in fp32
//      and write K^ as bf16 into a 128B-swizzled tile beside the v tile; one
//      thread issues tcgen05.mma (bf16, fp32 accumulation in TMEM).  The
//      Conv1D of v is linear, so it is folded into the contraction:
//      S = sum_tau w_tau (K^T v shifted by tau), the four shifted views of the
//      raw v tile forming one N = 256 operand, and the taps are applied per
//      column when the accumulators are drained.  The diagonal D x D blocks
//      are the segment's partial state; z, m and l = sum 2^a' complete its
//      record.
//  tc_reduce_kernel  fixed-order, max-rescaled combination of the records
//      into S = K^T V~ and z = K^T 1 with the softmax gate.
//  tc_readout_kernel (Sec. 2.1 item 2 readout and item 3)
//      Persistent; 128-token tiles of one (batch, head).  Eight producer warps
//      compute phi(Conv1D(q)) from a TMA q tile into a K-major bf16 tile; one
//      thread issues tcgen05.mma against [S | z] (bf16 hi + lo, N = D + 16),
//      giving phi(q~)^T S and phi(q~)^T z per token in TMEM; eight epilogue
//      warps (two per TMEM lane quarter, one token row per thread) divide,
//      apply RMSNorm, the norm weight and SiLU(out_gate) (out_gate tile
//      brought in by TMA) and write o in place of the out_gate tile, which TMA
//      stores back.
//
// Why V~ is never rounded to bf16: V~ = Conv1D(v) is not representable in
// bf16, and its rounding error does not average out, because O is a heavily
// cancelling weighted mean of the v rows (|O| shrinks like 1/sqrt(L) while the
// rows stay O(1)).  The state kernel multiplies the raw bf16 v (exact) and
// applies the fp32 taps to the fp32 accumulators; the readout multiplies by
// [S | z] as a bf16 hi + lo pair.  K^ only weights the mean, so bf16 is
// enough there.
//
// Every mbarrier wait is bounded (2 s).  A wait that runs out sets a bit in
// g_tc_error and the CTA's abort flag; the other waits then return at once,
// the roles run to the end of their loops without blocking (keeping named
// barriers matched), and the CTA frees its TMEM after its MMAs have drained.
#include <math.h>

#include <mutex>

#include "gbla_internal.cuh"
#include "gbla_sm100.cuh"

namespace gbla {

// Error word written by a kernel whose bounded wait ran out.
__device__ unsigned int g_tc_error;

namespace {

using namespace sm100;

constexpr int kGroupCh = 128;  // channels of one head group: MMA M and N of the state

// ------------------------------------------------------------------ state
// 19 warps: two groups of 8 converter warps, each group converting one
// 32-token half of every 64-token stage; one warp issues the MMAs; warp 17
// loads the k tiles (one issuing lane per k ring slot) and warp 18 the v tiles
// (two issuing lanes, lane l filling the v slots l and l + 2: a single
// issuing thread caps an SM's bulk-copy rate at about one box per 0.5 us,
// below its share of HBM bandwidth).  Every waiter on a ring barrier waits for
// each of its phases in turn (a parity wait can only tell the current phase
// from the one before it).
//
// The k tile of a stage (one head group, 64 tokens + 3 rows of conv history)
// lands in the k ring and is free again as soon as the converters have turned
// it into K^ = g phi(Conv1D(k)) (bf16, the A operand), which they write into
// the K^ ring.  The v tile (two 64-channel blocks, 128B-swizzled) lands in the
// v ring and is the B operand as it stands: the Conv1D of v is linear, so
// S = sum_tau w_tau (K^T v shifted by tau), the four shifted views of the v
// tile forming one N = 256 operand per block, with the taps applied per column
// when the accumulators are drained.  V~ is never formed or rounded.
constexpr int kSGroupWarps = 8;                      // converter warps per group
constexpr int kSCvtWarps = 2 * kSGroupWarps;         // 16
constexpr int kSMmaWarp = kSCvtWarps;                // 16
constexpr int kSKWarp = kSCvtWarps + 1;              // 17: k tiles
constexpr int kSVWarp = kSCvtWarps + 2;              // 18: v tiles
constexpr int kSThreads = (kSVWarp + 1) * 32;        // 608
constexpr int kSProd = kSCvtWarps * 32;              // converter threads
constexpr int kSTok = 64;                            // tokens per stage
constexpr int kSHalo = kConvW - 1;                   // conv history rows in front of a tile
constexpr int kSRawRows = kSTok + kSHalo;            // 67
constexpr int kSRawRowB = kGroupCh * 2;              // bytes of one token's k group row
constexpr int kSKBox = kSRawRows * kSRawRowB;        // 17152: one k tile
constexpr int kSKStages = 4;                         // k ring: one issuing lane per slot
constexpr int kSVBlock = 72 * 128;                   // 9216: v block pitch (1024-aligned)
constexpr int kSVBoxBytes = kSRawRows * 128;         // 8576 written by one v box
constexpr int kSMnBlock = kSTok * 128;               // 8192: one 64-channel MN block of K^
// The K^ tile only has to outlive its stage's MMAs, while the v tile is
// fetched stages ahead, so they have rings of their own: the shared memory a
// K^ slot per v slot would take goes to a deeper k ring (a per-stage clock64
// trace showed the converters waiting ~600 cycles a stage for their k tile
// with three k slots).
constexpr int kSKhStage = 2 * kSMnBlock;             // 16384: one K^ tile (two MN blocks)
constexpr int kSKhStages = 3;                        // K^ ring
constexpr int kSVStage = 2 * kSVBlock;               // 18432: one v tile (two blocks)
constexpr int kSVStages = 4;                         // v ring: v lane l fills l, l + 2
constexpr int kSVLanes = 2;
constexpr int kRangeStages = 32;                     // longest range (stages)
constexpr int kRangeTok = kRangeStages * kSTok;      // 2048
constexpr uint32_t kSTmemCols = 512;                 // per v block: 4 taps x 64 columns

constexpr int kMaxBatch = 2048;

// Shared-memory map of the state kernel (offsets from a 1024-aligned base).
constexpr int kSOffKh = 0;
constexpr int kSOffV = kSOffKh + kSKhStages * kSKhStage;
constexpr int kSOffK = kSOffV + kSVStages * kSVStage;
constexpr int kSOffGate = kSOffK + kSKStages * kSKBox;              // u16 [2][kRangeTok]
constexpr int kSOffHmax = kSOffGate + 2 * kRangeTok * 2;            // float [2][64]: half-stage max
constexpr int kSOffSegm = kSOffHmax + 2 * 64 * 4;                   // float [2][32]: segment max
constexpr int kSOffZred = kSOffSegm + 2 * kRangeStages * 4;         // float [16][128]
constexpr int kSOffLred = kSOffZred + 16 * kGroupCh * 4;            // float [16][2]
constexpr int kSOffWv = kSOffLred + 16 * 2 * 4;                     // float4 [128]: v taps
constexpr int kSOffRed = kSOffWv + kGroupCh * 16;                   // int [32]: scan scratch
constexpr int kSOffPre = kSOffRed + 32 * 4;                         // int [kMaxBatch + 1]
constexpr int kSOffBar = kSOffPre + ((kMaxBatch + 1) * 4 + 15) / 16 * 16;
// k_full, k_empty, kh_full (K^ written), kh_empty, v_full (v landed), v_empty,
// done, final, logits_in (the first range's gate logits are in shared memory)
constexpr int kSBarCount = 2 * kSKStages + 2 * kSKhStages + 2 * kSVStages + 3;
constexpr int kSOffMisc = kSOffBar + kSBarCount * 8;                // tmem addr, abort flag
constexpr int kSSmemBytes = kSOffMisc + 16 + 1024;                  // + alignment slack
static_assert(kSSmemBytes <= 227 * 1024, "state shared memory");
static_assert(kSKhStage % 1024 == 0 && kSVStage % 1024 == 0 && kSVBlock % 1024 == 0 &&
                  kSOffV % 1024 == 0 && kSOffK % 128 == 0 && kSKBox % 128 == 0,
              "TMA and swizzled operand alignment");
static_assert(kSVStages % kSVLanes == 0, "each v slot has one issuing lane");

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

// ------------------------------------------------------------------ readout
// 19 warps: 8 producer, 8 epilogue (two per TMEM lane quarter), MMA, and one
// TMA warp each for out_gate and q.  At most 5 warps per SM sub-partition, so
// each thread may hold 96 registers.
constexpr int kRTok = 128;                      // tokens per tile (MMA M)
constexpr int kRProdWarps = 8;
constexpr int kREpiWarps = 8;
constexpr int kRMmaWarp = kRProdWarps + kREpiWarps;   // 16
constexpr int kRTmaWarp = kRMmaWarp + 1;              // 17: out_gate loads
constexpr int kRQWarp = kRTmaWarp + 1;                // 18: q loads
constexpr int kRThreads = (kRQWarp + 1) * 32;         // 608
constexpr int kRProd = kRProdWarps * 32;
constexpr int kREpi = kREpiWarps * 32;
constexpr int kRAStages = 2;
constexpr int kRAccBufs = 2;
constexpr int kRQRows = kRTok + 3;              // q tile rows: 3-token conv halo + tile

template <int D>
struct ReadoutCfg {
  static constexpr bool QT = D == 64;                     // q through TMA into its own ring
  // D = 128: no room for a q ring beside [S | z] (N = 144, hi + lo) and the
  // out_gate stages, so q comes by TMA straight into the A slot (3 rows of
  // conv history in front) and the producers turn it into phi(Conv1D(q)) in
  // place; the MMA reads the slot from row 3 on.
  static constexpr bool QA = D == 128;
  static constexpr int NR = D + 16;                       // MMA N: D columns of S, z, zeros
  static constexpr int KB = D / 64;                       // 64-element K blocks
  static constexpr int NCH = QT ? 4 : 8;                  // channels per producer thread
  static constexpr int TPR = D / NCH;                     // producer threads per token row
  static constexpr int STREAMS = kRProd / TPR;            // producer sub-streams per tile
  static constexpr int TPS = kRTok / STREAMS;             // tokens per sub-stream
  // one 64-channel block of an A slot: 128 token rows (QA: 131 with the conv
  // history, rounded up to whole 1024-byte swizzle atoms)
  static constexpr int kABlk = QA ? (kRQRows * 128 + 1023) / 1024 * 1024 : kRTok * 128;
  static constexpr int kARow0 = QA ? 3 * 128 : 0;          // byte offset of A row 0 in a block
  static constexpr int kABytes = KB * kABlk;              // one A slot
  static constexpr int kBBytes = NR * D * 2;              // one of B_hi / B_lo
  static constexpr int kOgStages = D == 128 ? 2 : 4;
  static constexpr int kOgBytes = kRTok * D * 2;
  static constexpr int kQStages = QT ? 3 : (QA ? kRAStages : 0);  // QA: one per A slot
  static constexpr int kQTileBytes = kRQRows * 128;                  // one 64-channel block
  static constexpr int kQBytes = (kQTileBytes + 1023) / 1024 * 1024;  // 1024-aligned stride
  static constexpr int kOffA = 0;
  static constexpr int kOffBhi = kOffA + kRAStages * kABytes;
  static constexpr int kOffBlo = kOffBhi + kBBytes;
  static constexpr int kOffOg = kOffBlo + kBBytes;
  static constexpr int kOffQ = kOffOg + kOgStages * kOgBytes;
  static constexpr int kOffPre = kOffQ + (QT ? kQStages * kQBytes : 0);  // int [kMaxBatch + 1]
  static constexpr int kOffSs = kOffPre + ((kMaxBatch + 1) * 4 + 15) / 16 * 16;  // float [256]
  static constexpr int kOffW = kOffSs + kREpi * 4;  // float [D]: norm weights of the head
  static constexpr int kOffBar = kOffW + D * 4;
  // a_full[2], a_empty[2], og_full[S], og_empty[S], q_full[Q], q_empty[Q],
  // acc_full[2], acc_empty[2], b_full, b_free, final
  static constexpr int kBars =
      2 * kRAStages + 2 * kOgStages + 2 * kQStages + 2 * kRAccBufs + 3;
  static constexpr int kOffMisc = kOffBar + kBars * 8;
  static constexpr int kSmem = kOffMisc + 16 + 1024;
  static constexpr uint32_t kAccStride = NR <= 128 ? 128 : 256;  // column offset of buffer 1
  static constexpr uint32_t kTmemCols = kAccStride + NR <= 256 ? 256 : 512;
  static constexpr uint32_t kIdesc = idesc_bf16_f32(kRTok, NR, 0, 0);
  static_assert(kSmem <= 227 * 1024, "readout shared memory");
  static_assert(TPS % 4 == 0, "producer sub-streams are processed 4 tokens at a time");
  static_assert(!QT || TPS == 8, "TMA q path: one 8-row swizzle atom per sub-stream");
};

__device__ __forceinline__ void report_error(unsigned code, const AbortFlag &ab) {
  atomicOr(&g_tc_error, code);
  ab.raise();
}

__device__ __forceinline__ int clamp_len(const int32_t *seq_lens, int b, int N) {
  if (seq_lens == nullptr) return N;
  int L = seq_lens[b];
  return L < 0 ? 0 : (L > N ? N : L);
}

// Exclusive prefix over b of count(b) into pre[0..B], computed by the `nthr`
// threads with tid < nthr (a multiple of 32, at most 1024).  Ends with a named
// barrier over those threads.
template <typename CountFn>
__device__ void prefix_counts(int *pre, int B, int tid, int nthr, uint32_t bar_id,
                              int *warp_tot, CountFn count) {
  const int per = (B + nthr - 1) / nthr;
  const int lo = min(B, tid * per), hi = min(B, lo + per);
  int s = 0;
  for (int i = lo; i < hi; ++i) s += count(i);
  const int lane = tid & 31, warp = tid >> 5;
  int x = s;  // inclusive warp scan
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_tot[warp] = x;
  named_barrier(bar_id, nthr);
  int off = 0;
  for (int w = 0; w < warp; ++w) off += warp_tot[w];
  int run = off + x - s;  // exclusive start of this thread's segment
  if (tid == 0) pre[0] = 0;
  for (int i = lo; i < hi; ++i) {
    run += count(i);
    pre[i + 1] = run;
  }
  named_barrier(bar_id, nthr);
}

// Largest b with pre[b] <= k (pre nondecreasing, pre[0] = 0 <= k < pre[B]).
__device__ __forceinline__ int find_batch(const int *pre, int B, int k) {
  int lo = 0, hi = B;  // invariant: pre[lo] <= k < pre[hi]
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (pre[mid] <= k) lo = mid; else hi = mid;
  }
  return lo;
}

__device__ __forceinline__ void unpack8(const uint4 &r, float (&x)[8]) {
  const uint32_t w[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 f = bf2_to_f2(w[i]);
    x[2 * i] = f.x;
    x[2 * i + 1] = f.y;
  }
}
__device__ __forceinline__ void unpack4(const uint2 &r, float (&x)[4]) {
  const float2 a = bf2_to_f2(r.x), b = bf2_to_f2(r.y);
  x[0] = a.x; x[1] = a.y; x[2] = b.x; x[3] = b.y;
}

// Causal Conv1D of channels i, i+1: taps 0..2 on x[t-3..t-1], tap 3 on x[t].
template <int NC>
__device__ __forceinline__ float2 conv2(const float (&w)[4][NC], const float (&xm)[3][NC],
                                        const float (&x)[NC], int i) {
  float2 a = __fmul2_rn(make_float2(w[0][i], w[0][i + 1]), make_float2(xm[0][i], xm[0][i + 1]));
  a = __ffma2_rn(make_float2(w[1][i], w[1][i + 1]), make_float2(xm[1][i], xm[1][i + 1]), a);
  a = __ffma2_rn(make_float2(w[2][i], w[2][i + 1]), make_float2(xm[2][i], xm[2][i + 1]), a);
  a = __ffma2_rn(make_float2(w[3][i], w[3][i + 1]), make_float2(x[i], x[i + 1]), a);
  return a;
}

template <int NC>
__device__ __forceinline__ void slide(float (&xm)[3][NC], const float (&x)[NC]) {
#pragma unroll
  for (int i = 0; i < NC; ++i) {
    xm[0][i] = xm[1][i];
    xm[1][i] = xm[2][i];
    xm[2][i] = x[i];
  }
}

// phi(x) = elu(x) + 1 for two channels given xl = x * log2(e):
// exp(min(x, 0)) + max(x, 0) = 2^mn + ln2 (xl - mn),  mn = min(xl, 0).
__device__ __forceinline__ float2 phi2_log2(float2 xl) {
  const float2 mn = make_float2(fminf(xl.x, 0.f), fminf(xl.y, 0.f));
  const float2 e = make_float2(ex2_approx(mn.x), ex2_approx(mn.y));
  const float2 d = __ffma2_rn(mn, make_float2(-1.f, -1.f), xl);
  return __ffma2_rn(make_float2(kLn2, kLn2), d, e);
}

// Causal Conv1D of channels i, i+1 at token u of a thread's 4 tokens: taps
// 0..3 on raw rows u..u+3 (row u + 3 is the token itself).
__device__ __forceinline__ float2 conv_rows(const float (&w)[4][4], const float (&x)[7][4],
                                            int u, int i) {
  float2 a = __fmul2_rn(make_float2(w[0][i], w[0][i + 1]), make_float2(x[u][i], x[u][i + 1]));
#pragma unroll
  for (int tau = 1; tau < 4; ++tau)
    a = __ffma2_rn(make_float2(w[tau][i], w[tau][i + 1]),
                   make_float2(x[u + tau][i], x[u + tau][i + 1]), a);
  return a;
}

// Causal Conv1D of channels i, i+1 at row u + 3 of a row array: taps 0..3 on
// rows u..u+3.
template <int R>
__device__ __forceinline__ float2 conv_rows_n(const float (&w)[4][4], const float (&x)[R][4],
                                              int u, int i) {
  float2 a = __fmul2_rn(make_float2(w[0][i], w[0][i + 1]), make_float2(x[u][i], x[u][i + 1]));
#pragma unroll
  for (int tau = 1; tau < 4; ++tau)
    a = __ffma2_rn(make_float2(w[tau][i], w[tau][i + 1]),
                   make_float2(x[u + tau][i], x[u + tau][i + 1]), a);
  return a;
}

// K^ of two channels from x' = k~ log2(e) and the token's a' = (a - m) log2(e),
// wl = 2^a' ln 2:  K^ = 2^a' phi(k~) = wl (x' - min(x', 0)) + 2^(min(x', 0) + a').
__device__ __forceinline__ float2 khat2(float2 xl, float al, float wl) {
  const float2 mn = make_float2(fminf(xl.x, 0.f), fminf(xl.y, 0.f));
  const float2 d = __ffma2_rn(mn, make_float2(-1.f, -1.f), xl);
  const float2 ea = __fadd2_rn(mn, make_float2(al, al));
  const float2 e = make_float2(ex2_approx(ea.x), ex2_approx(ea.y));
  return __ffma2_rn(make_float2(wl, wl), d, e);
}

__device__ __forceinline__ float bf16_bits_to_f32(unsigned short r) {
  return __uint_as_float((uint32_t)r << 16);
}

// a' = (a - m) log2(e) of a gate logit given as bf16 bits, with mlog = m log2(e)
// (0 when the head is missing: its logits are all -inf, and so is a').
__device__ __forceinline__ float gate_log2(unsigned short a, float mlog) {
  return fmaf(__uint_as_float((uint32_t)a << 16), kLog2e, -mlog);
}

// One token quad of a converter thread, k side: channels 4q..4q+3 of the head
// group at 4 consecutive tokens of the stage.  Reads the 7 raw k rows it needs
// (3 of conv history) from the TMA tile and the 4 tokens' gate logits,
// convolves, applies phi and the gate weight, and writes K^ as bf16 into the
// MN-major, 128B-swizzled A tile (one 8-byte piece per token row).  Tokens past
// the sequence end (nvalid < 4) are zeros.  Returns the sum of 2^a' ln 2 over
// the 4 tokens (0 for tokens past the end, whose logits are -inf).
// FULL: all 4 tokens are valid (nvalid == 4), the case of every token quad but
// the sequence's last, compiled without the masking.
template <bool FULL>
__device__ __forceinline__ float state_convert_k(uint32_t raw, uint32_t arow, uint32_t cs,
                                                 uint32_t gws, float mlog, const float (&w)[4][4],
                                                 float2 (&z)[2], int nvalid) {
  float x[7][4];
#pragma unroll
  for (int r = 0; r < 7; ++r) unpack4(lds_v2(raw + r * kSRawRowB), x[r]);
  const uint2 g4 = lds_v2(gws);  // 4 bf16 logits
  const unsigned short ga[4] = {(unsigned short)(g4.x & 0xffffu), (unsigned short)(g4.x >> 16),
                                (unsigned short)(g4.y & 0xffffu), (unsigned short)(g4.y >> 16)};
  float lsum = 0.f;
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const float al = gate_log2(ga[u], mlog), wl = ex2_approx(al) * kLn2;
    lsum += wl;
    float2 k01 = khat2(conv_rows(w, x, u, 0), al, wl);
    float2 k23 = khat2(conv_rows(w, x, u, 2), al, wl);
    if (!FULL && u >= nvalid) {  // rows past the sequence end may hold anything, NaN included
      k01 = make_float2(0.f, 0.f);
      k23 = make_float2(0.f, 0.f);
    }
    z[0] = __fadd2_rn(z[0], k01);
    z[1] = __fadd2_rn(z[1], k23);
    sts_v2(arow + u * 128 + ((cs ^ u) << 4), f2_to_bf2(k01.x, k01.y), f2_to_bf2(k23.x, k23.y));
  }
  return lsum;
}

// ===================================================================== state
struct StateParams {
  const __nv_bfloat16 *gate;
  const float *conv_w;
  const int32_t *seq_lens;
  float *records;        // [ranges + sequences][G][D*D + D + 4]: S as [c / 8][a][c % 8], z, m, l, 2 pad
  int B, H, N, HG;
  uint32_t flags;        // gbla_flags (NO_CONV, NO_GATE)
};

// Work split.  The state step's work is the list of 64-token stages of all
// (batch, head group) sequences in (batch, head group, token) order, NS
// stages in all.  It is cut into R balanced ranges of consecutive stages, R a
// multiple of the grid size P chosen so that no range is longer than
// kRangeStages; CTA x takes ranges x, x + P, ...  A range may span several
// sequences; its part in one sequence is a segment, and each segment leaves one
// partial record (S, z and the gate's m, l over the segment).  Sequence q and
// range r meet in at most one segment, stored as record q + r: for q < q' every
// range meeting q comes no later than every range meeting q', so the index is
// unique, and below R + Q (Q sequences).
__host__ __device__ __forceinline__ long long num_ranges(long long NS, long long P) {
  return NS <= 0 ? 0 : P * ((NS + kRangeStages * P - 1) / (kRangeStages * P));
}
__device__ __forceinline__ long long range_begin(long long NS, long long R, long long r) {
  return NS * r / R;
}
// The range holding stage s, the largest r with range_begin(r) <= s, i.e.
// floor(((s + 1) R - 1) / NS), without a 64-bit division: a double-precision
// estimate corrected by exact integer products.
__device__ __forceinline__ long long range_of(long long NS, long long R, long long s) {
  const long long x = (s + 1) * R - 1;
  long long r = (long long)((double)x / (double)NS);
  while (r > 0 && r * NS > x) --r;
  while ((r + 1) * NS <= x) ++r;
  return r;
}

// The sequence of stage s: batch b, head group hg, stage st of its nst stages
// (L tokens); s0 is the sequence's first stage in the flattened list.
struct StageRef {
  int b, hg, st, nst, L;
  long long s0;
};
// Stage indices fit in 32 bits (at most 2^30 stages, checked on the host).
__device__ __forceinline__ StageRef decode_stage(const StateParams &p, const int *pre,
                                                 long long s64) {
  StageRef r;
  const int s = (int)s64;
  if (p.seq_lens == nullptr) {  // every sequence has N tokens: arithmetic only
    r.L = p.N;
    r.nst = (p.N + kSTok - 1) / kSTok;
    const int per_b = p.HG * r.nst;
    r.b = s / per_b;
    const int rem = s - r.b * per_b;
    r.hg = rem / r.nst;
    r.st = rem - r.hg * r.nst;
  } else {
    r.b = find_batch(pre, p.B, s);
    r.L = clamp_len(p.seq_lens, r.b, p.N);
    r.nst = (r.L + kSTok - 1) / kSTok;
    const int rem = s - pre[r.b];
    r.hg = rem / r.nst;
    r.st = rem - r.hg * r.nst;
  }
  r.s0 = s64 - r.st;
  return r;
}

// ABL: the ablation instantiation, which reads p.flags; the default one
// compiles the full core with no flag tests.
template <int D, bool ABL>
__global__ void __launch_bounds__(kSThreads, 1)
    tc_state_kernel(const StateParams p, const __grid_constant__ CUtensorMap tm_k,
                    const __grid_constant__ CUtensorMap tm_v) {
  constexpr int G = kGroupCh / D;
  constexpr int REC = D * D + D + 4;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  unsigned short *gw = (unsigned short *)(smem + kSOffGate);  // [2][kRangeTok]: logits
  float *hmax = (float *)(smem + kSOffHmax);  // [2][64]: half-stage maxima of the range
  float *segm = (float *)(smem + kSOffSegm);  // [2][32]: max over each stage's segment
  float *zred = (float *)(smem + kSOffZred);  // [16][128]
  float *lred = (float *)(smem + kSOffLred);  // [16][2]
  float4 *wvs = (float4 *)(smem + kSOffWv);   // [128]: v taps of the group's channels
  int *pre = (int *)(smem + kSOffPre);
  uint64_t *bars = (uint64_t *)(smem + kSOffBar);
  uint64_t *k_full = bars, *k_empty = bars + kSKStages;
  uint64_t *kh_full = bars + 2 * kSKStages, *kh_empty = kh_full + kSKhStages;
  uint64_t *v_full = kh_empty + kSKhStages, *v_empty = v_full + kSVStages;
  uint64_t *done = v_empty + kSVStages, *fin = done + 1, *logits_in = fin + 1;
  uint32_t *tmem_slot = (uint32_t *)(smem + kSOffMisc);
  const AbortFlag ab{smem_u32(smem + kSOffMisc + 4)};

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int B = p.B, H = p.H;
  const uint32_t flags = ABL ? p.flags : 0u;

  // Converter thread -> (group, channel quad q, token quad j): group grp takes
  // token rows 32 grp .. 32 grp + 31 of every stage; within a group the mapping
  // makes both the raw-tile reads (16 lanes, 16 distinct quads of one 256-byte
  // row) and the swizzled K^ writes (16 lanes, 16 distinct 8-byte slots of the
  // 128-byte bank window) free of bank conflicts.
  const int grp = warp / kSGroupWarps;
  const int hw = 2 * (warp % kSGroupWarps) + (lane >> 4);              // half-warp 0..15
  const int q = (lane & 15) + 16 * (hw & 1);                           // channel quad 0..31
  const int j = (((lane >> 1) & 3) ^ (hw >> 2)) + 4 * ((hw >> 1) & 1);  // token quad 0..7
  const int c0ch = 4 * q;
  const int hh = c0ch / D, d0 = c0ch - D * hh;                         // head in group, channel

  if (tid == 0) {
    *(volatile int *)(smem + kSOffMisc + 4) = 0;
    for (int i = 0; i < kSKStages; ++i) {
      mbar_init(&k_full[i], 1);            // the k box (expect_tx)
      mbar_init(&k_empty[i], kSCvtWarps);  // released by both converter groups
    }
    for (int i = 0; i < kSKhStages; ++i) {
      mbar_init(&kh_full[i], kSCvtWarps);  // K^ written (and v rows past the end zeroed)
      mbar_init(&kh_empty[i], 1);          // the stage's MMAs completed
    }
    for (int i = 0; i < kSVStages; ++i) {
      mbar_init(&v_full[i], 1);            // the v boxes (expect_tx)
      mbar_init(&v_empty[i], 1);           // the stage's MMAs completed
    }
    mbar_init(done, 1);
    mbar_init(fin, 1);
    mbar_init(logits_in, kSCvtWarps);
    fence_mbar_init();
  }
  if (warp == kSKWarp && lane == 0) {
    tma_prefetch_desc(&tm_k);
    tma_prefetch_desc(&tm_v);
  }
  __syncthreads();
  // The grid is launched with programmatic dependent launch: the set-up above
  // overlaps the end of the kernel before it on the stream, whose results the
  // inputs may be; nothing is read before that kernel has completed, and the
  // dependents (the reduction) launch only after this wait.
  grid_dep_wait();

  // Stage prefix over the batch (ragged lengths only; uniform lengths decode
  // by arithmetic, so the first loads go out at once).
  long long NS;
  if (p.seq_lens == nullptr) {
    NS = (long long)B * p.HG * ((p.N + kSTok - 1) / kSTok);
  } else {
    if (warp < kSCvtWarps)
      prefix_counts(pre, B, tid, kSProd, 1, (int *)(smem + kSOffRed), [&](int b) {
        const int L = clamp_len(p.seq_lens, b, p.N);
        return p.HG * ((L + kSTok - 1) / kSTok);
      });
    __syncthreads();
    NS = pre[B];
  }
  const long long R = num_ranges(NS, gridDim.x);
  grid_dep_launch();
  if ((long long)blockIdx.x >= R) return;  // no work for this CTA

  if (warp >= kSKWarp) {
    // ------------------------------------------------------------ TMA loads
    // Warp 17: the k tile of each stage (one head group x 67 token rows, no
    // swizzle; lane l issues the stages whose index in the CTA's stage
    // sequence is l mod 3, all into k slot l).  Warp 18: the v tile (two
    // 64-channel blocks x 67 rows, 128B swizzle) into the stage's operand slot
    // (lane l issues the stages with index l mod 2, operand slots l and l + 2).
    // 3 rows of conv history in front, zero-filled before the sequence start.
    // Only the CTA's first stage goes out before the converters' gate logits of
    // its first range are in shared memory (mbarrier logits_in): the logits
    // would otherwise queue behind the start-up burst of every CTA's copies.
    const bool kw = warp == kSKWarp;
    const int nl = kw ? kSKStages : kSVLanes;
    const uint64_t pol = l2_policy_evict_first();
    auto issue = [&](long long s, uint32_t gs) -> bool {
      const StageRef st = decode_stage(p, pre, s);
      const int tok = st.st * kSTok - kSHalo;
      if (kw) {
        const uint32_t ks = gs % kSKStages, ph = (gs / kSKStages) & 1;
        if (!mbar_wait(&k_empty[ks], ph ^ 1, &ab)) return false;
        mbar_arrive_expect_tx(&k_full[ks], kSKBox);
        tma_load_4d_hint(smem + kSOffK + ks * kSKBox, &tm_k, &k_full[ks], 0, st.hg * G, tok, st.b,
                         pol);
      } else {
        const uint32_t os = gs % kSVStages, ph = (gs / kSVStages) & 1;
        if (!mbar_wait(&v_empty[os], ph ^ 1, &ab)) return false;
        uint8_t *dst = smem + kSOffV + os * kSVStage;
        // the second block is absent for a missing head (D = 64, odd H)
        const bool two = !(D == 64 && st.hg * G + 1 >= H);
        mbar_arrive_expect_tx(&v_full[os], (two ? 2 : 1) * kSVBoxBytes);
        for (int blk = 0; blk < (two ? 2 : 1); ++blk)
          tma_load_4d_hint(dst + blk * kSVBlock, &tm_v, &v_full[os], (blk * 64) % D,
                           st.hg * G + (blk * 64) / D, tok, st.b, pol);
      }
      return true;
    };
    uint32_t last = 0xffffffffu;
    bool ok = true;
    const long long s_first = range_begin(NS, R, blockIdx.x);
    if (lane == 0 && s_first < range_begin(NS, R, blockIdx.x + 1)) {  // a non-empty first range
      ok = issue(s_first, 0);
      if (ok) last = 0;
    }
    if (lane < nl) {
      if (!mbar_wait(logits_in, 0, &ab)) ok = false;
      uint32_t gs = 0;
      for (long long r = blockIdx.x; r < R && ok; r += gridDim.x) {
        const long long se = range_begin(NS, R, r + 1);
        for (long long s = range_begin(NS, R, r); s < se; ++s, ++gs) {
          if (gs == 0 || gs % nl != (uint32_t)lane) continue;  // stage 0 went out above
          if (!issue(s, gs)) {
            ok = false;
            break;
          }
          last = gs;
        }
      }
      if (!ok && !ab.raised()) report_error(2048, ab);
      // every copy this lane issued has landed before the CTA can exit (the
      // phases of its slot complete in order: waiting for the last suffices)
      if (last != 0xffffffffu) {
        const bool okw = kw ? mbar_wait(&k_full[last % kSKStages], (last / kSKStages) & 1, nullptr)
                            : mbar_wait(&v_full[last % kSVStages], (last / kSVStages) & 1, nullptr);
        if (!okw) report_error(4096, ab);
      }
    }
    __syncthreads();
    return;
  }

  // TMEM hand-off between the MMA warp and the converters (barrier 2); the
  // converters join it after the first range's gate pre-pass.
  uint32_t tmem = 0;
  auto tmem_handoff = [&]() {
    tc_fence_before();
    named_barrier(2, kSProd + 32);
    tc_fence_after();
    tmem = *tmem_slot;
  };

  if (warp < kSCvtWarps) {
    // ------------------------------------------------------------ converters
    // K^ rows: MN block q / 16, token row 4j + u, 16-byte chunk (q % 16) / 2
    // swizzled by the row, 8-byte half q & 1
    const uint32_t arow0 = smem_u32(smem + kSOffKh) +
                           (uint32_t)((q >> 4) * kSMnBlock + 4 * j * 128 + (q & 1) * 8);
    const uint32_t cs = (uint32_t)(((q & 15) >> 1) ^ (4 * (j & 1)));
    const uint32_t raw0 = smem_u32(smem + kSOffK) + (uint32_t)(4 * j * kSRawRowB + q * 8);
    const uint32_t gws = smem_u32(gw) + (uint32_t)(hh * kRangeTok + 4 * j) * 2;
    const bool no_conv = flags & GBLA_FLAG_NO_CONV, no_gate = flags & GBLA_FLAG_NO_GATE;
    uint32_t gs0 = 0;  // first stage of the segment in the CTA's stage sequence
    int nseg = 0, cur_hg = -1;
    float wk[4][4];    // k taps of this thread's channels, times log2 e
    bool first = true;
    for (long long r = blockIdx.x; r < R; r += gridDim.x) {
      const long long sb = range_begin(NS, R, r), se = range_begin(NS, R, r + 1);
      const int nsr = (int)(se - sb);
      // ---- range pre-pass: the range's gate logits into shared memory (-inf
      // past a sequence end or for a missing head), half-stage maxima, then
      // for every stage the maximum over its segment.
      {
        // For each i, the 32 slots tid + i kSProd of a warp are 32 consecutive
        // tokens of one stage: lane i decodes the warp's stage for that i, and
        // each stage's (b, hg, stage, L) reaches the other lanes by shuffle, so
        // the decodes (a search of the stage prefix and a length load when
        // ragged) run side by side.
        constexpr int NSL = kRangeTok / kSProd;
        static_assert(kSTok % 32 == 0 && kSProd % 32 == 0 && NSL <= 32,
                      "a warp's 32 slots for one i lie in one stage");
        int db = 0, dhg = 0, dst = 0, dL = 0;
        if (lane < NSL && (tid & ~31) + lane * kSProd < nsr * kSTok) {
          const StageRef st = decode_stage(p, pre, sb + ((tid & ~31) + lane * kSProd) / kSTok);
          db = st.b;
          dhg = st.hg;
          dst = st.st;
          dL = st.L;
        }
        unsigned short a[NSL][G];
#pragma unroll
        for (int i = 0; i < NSL; ++i) {
          const int slot = tid + i * kSProd;
          const int sbi = __shfl_sync(0xffffffffu, db, i), shg = __shfl_sync(0xffffffffu, dhg, i);
          const int sst = __shfl_sync(0xffffffffu, dst, i), sL = __shfl_sync(0xffffffffu, dL, i);
#pragma unroll
          for (int g = 0; g < G; ++g) a[i][g] = 0xff80u;  // bf16 -inf
          if (slot < nsr * kSTok) {
            const int t = sst * kSTok + slot % kSTok;
            if (t < sL) {
              const unsigned short *gp = (const unsigned short *)p.gate +
                                         ((size_t)sbi * p.N + t) * H + shg * G;
#pragma unroll
              for (int g = 0; g < G; ++g)
                if (shg * G + g < H) a[i][g] = no_gate ? (unsigned short)0 : __ldg(gp + g);
            }
          }
        }
#pragma unroll
        for (int i = 0; i < NSL; ++i) {
          const int slot = tid + i * kSProd;
#pragma unroll
          for (int g = 0; g < G; ++g) {
            gw[g * kRangeTok + slot] = a[i][g];
            float m = bf16_bits_to_f32(a[i][g]);
#pragma unroll
            for (int o = 16; o >= 1; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
            if (lane == 0) hmax[g * 64 + slot / 32] = m;
          }
        }
        if (first) {  // logits in: the TMA warps go on
          __syncwarp();
          if (lane == 0) mbar_arrive(logits_in);
        }
        named_barrier(1, kSProd);
        if (tid < G * 32) {
          const int g = tid / 32, k = tid % 32;
          if (k < nsr) {
            const StageRef st = decode_stage(p, pre, sb + k);
            const int k0 = (int)(max(sb, st.s0) - sb), k1 = (int)(min(se, st.s0 + st.nst) - sb);
            float m = -INFINITY;
            for (int i = k0; i < k1; ++i)
              m = fmaxf(m, fmaxf(hmax[g * 64 + 2 * i], hmax[g * 64 + 2 * i + 1]));
            segm[g * kRangeStages + k] = m;
          }
        }
        named_barrier(1, kSProd);
      }
      if (first) tmem_handoff();
      first = false;

      for (long long s = sb; s < se;) {
        const StageRef st = decode_stage(p, pre, s);
        const long long seg_end = min(se, st.s0 + st.nst);
        const int nst = (int)(seg_end - s), lst0 = (int)(s - sb);
        if (st.hg != cur_hg) {  // taps of this thread's 4 channels (identity: ablation)
          const int h = st.hg * G + hh;
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            float4 tk = make_float4(0.f, 0.f, 0.f, h < H ? 1.f : 0.f);
            if (h < H && !no_conv)
              tk = __ldg((const float4 *)(p.conv_w + ((size_t)(H + h) * D + d0 + i) * 4));
            wk[0][i] = tk.x * kLog2e;
            wk[1][i] = tk.y * kLog2e;
            wk[2][i] = tk.z * kLog2e;
            wk[3][i] = tk.w * kLog2e;
          }
          if (tid < kGroupCh) {  // v taps of group channel tid, applied at the drain
            const int hz = st.hg * G + tid / D, dz = tid % D;
            float4 tv = make_float4(0.f, 0.f, 0.f, hz < H ? 1.f : 0.f);
            if (hz < H && !no_conv)
              tv = __ldg((const float4 *)(p.conv_w + ((size_t)(2 * H + hz) * D + dz) * 4));
            wvs[tid] = tv;
          }
          cur_hg = st.hg;
        }
        // a missing head has only -inf logits: M = -inf, and a' = -inf with mlog 0
        const float M = segm[hh * kRangeStages + lst0];
        const float mlog = M == -INFINITY ? 0.f : M * kLog2e;
        float2 z[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
        float lacc = 0.f;
        for (int it = 0; it < nst; ++it) {  // this group converts token rows 32 grp .. 32 grp + 31
          const uint32_t gs = gs0 + it;
          const uint32_t ks = gs % kSKStages, kph = (gs / kSKStages) & 1;
          const uint32_t hs = gs % kSKhStages, hph = (gs / kSKhStages) & 1;
          const uint32_t os = gs % kSVStages, oph = (gs / kSVStages) & 1;
          if (!mbar_wait(&k_full[ks], kph, &ab) && !ab.raised()) report_error(1, ab);
          if (!mbar_wait(&kh_empty[hs], hph ^ 1, &ab) && !ab.raised()) report_error(1, ab);
          const int T = (st.st + it) * kSTok;
          const int nvalid = min(max(st.L - (T + 32 * grp + 4 * j), 0), 4);
          const uint32_t rawp = raw0 + ks * kSKBox + grp * 32 * kSRawRowB;
          const uint32_t arp = arow0 + hs * kSKhStage + grp * 32 * 128;
          const uint32_t gwp = gws + (uint32_t)((lst0 + it) * kSTok + 32 * grp) * 2;
          const float ls = nvalid == 4
                               ? state_convert_k<true>(rawp, arp, cs, gwp, mlog, wk, z, 4)
                               : state_convert_k<false>(rawp, arp, cs, gwp, mlog, wk, z, nvalid);
          if (d0 == 0) lacc += ls;
          __syncwarp();
          if (lane == 0) mbar_arrive(&k_empty[ks]);  // the k tile is consumed
          if (T + kSTok > st.L) {
            // v rows past the sequence end meet K^ = 0 in the MMA, but may hold
            // NaN or inf: zero them (both 64-channel blocks) once they have landed
            if (!mbar_wait(&v_full[os], oph, &ab) && !ab.raised()) report_error(1, ab);
            const int r0 = max(st.L - (T - kSHalo), 0);
            const uint32_t vb = smem_u32(smem + kSOffV) + os * kSVStage;
            for (int e = tid; e < (kSRawRows - r0) * 16; e += kSProd) {
              const int rr = r0 + e / 16, blk = (e / 8) & 1, ck = e & 7;
              sts_v4(vb + blk * kSVBlock + rr * 128 + ck * 16, make_uint4(0, 0, 0, 0));
            }
          }
          fence_proxy_async_smem();  // K^ (and zeroed v rows) visible to the tensor cores
          __syncwarp();
          if (lane == 0) mbar_arrive(&kh_full[hs]);
        }
        gs0 += nst;

        // ---- segment end: z and l (token quads of both groups summed in a
        // fixed order); S[a][c] = sum_tau w_tau[c] P_tau[a][c] on the diagonal
        // D x D blocks, P_tau of v channel c = 64 blk + c' in TMEM column
        // 256 blk + 64 tau + c'.
        *(float4 *)&zred[(grp * 8 + j) * kGroupCh + c0ch] = make_float4(z[0].x, z[0].y, z[1].x, z[1].y);
        if (d0 == 0) lred[(grp * 8 + j) * 2 + hh] = lacc;
        named_barrier(1, kSProd);
        if (!mbar_wait(done, nseg & 1, &ab) && !ab.raised()) report_error(2, ab);
        tc_fence_after();
        const long long rec = (long long)(st.b * p.HG + st.hg) + r;
        {
          constexpr int CPW = D / 4;                    // columns per warp
          const int q4 = warp & 3, part = warp >> 2;    // lane quarter, column quarter
          const int ch = 32 * q4 + lane;                // TMEM lane = group channel (row of S)
          const int ha = ch / D, d = ch - D * ha;
          const bool ok2 = st.hg * G + ha < H;
          const int cv0 = D * ha + part * CPW;          // first v channel (of the group)
          const uint32_t tl = tmem + ((uint32_t)(32 * q4) << 16) +
                              (uint32_t)(256 * (cv0 / 64) + cv0 % 64);
          // record layout of S: [c / 8][a][c % 8], so that a warp's stores of
          // 32 rows x 8 columns are one contiguous kilobyte
          float *dst = p.records + ((size_t)rec * G + ha) * REC + (size_t)(part * CPW / 8) * (D * 8) +
                       (size_t)d * 8;
#pragma unroll
          for (int cb = 0; cb < CPW; cb += 8) {
            float v0[8], v1[8], v2[8], v3[8];
            tmem_ld8(tl + cb, v0);
            tmem_ld8(tl + 64 + cb, v1);
            tmem_ld8(tl + 128 + cb, v2);
            tmem_ld8(tl + 192 + cb, v3);
            tmem_ld_wait_regs(v0);
            tmem_pin(v1);
            tmem_pin(v2);
            tmem_pin(v3);
            float o[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
              const float4 wt = wvs[cv0 + cb + i];
              o[i] = fmaf(wt.w, v3[i], fmaf(wt.z, v2[i], fmaf(wt.y, v1[i], wt.x * v0[i])));
            }
            if (ok2) {
              float4 *dq = (float4 *)(dst + (size_t)(cb / 8) * (D * 8));
              dq[0] = make_float4(o[0], o[1], o[2], o[3]);
              dq[1] = make_float4(o[4], o[5], o[6], o[7]);
            }
          }
        }
        if (tid < kGroupCh) {
          const int hz = tid / D, dz = tid - D * hz;
          if (st.hg * G + hz < H) {
            float zsum = 0.f;
            for (int jj = 0; jj < 16; ++jj) zsum += zred[jj * kGroupCh + tid];
            float *rz = p.records + ((size_t)rec * G + hz) * REC;
            rz[D * D + dz] = zsum;
            if (dz == 0) {
              float lt = 0.f;
              for (int jj = 0; jj < 16; ++jj) lt += lred[jj * 2 + hz];
              rz[D * D + D] = segm[hz * kRangeStages + lst0];
              rz[D * D + D + 1] = lt * (1.f / kLn2);
            }
          }
        }
        tc_fence_before();
        named_barrier(1, kSProd);  // drained before the next segment's MMAs, taps and z/l sums
        ++nseg;
        s = seg_end;
      }
    }
  } else if (warp == kSMmaWarp) {
    tmem_alloc(tmem_slot, kSTmemCols);
    tmem_handoff();
    if (lane == 0) {
      // ---------------------------------------------------------- MMA issuer
      // P_tau += K^T v[t - 3 + tau] for tau = 0..3 in one N = 256 MMA per
      // 64-channel v block: its four 64-column B blocks are the same v tile
      // with the start moved down 0..3 rows (LBO = one 128-byte row).  The
      // 128-byte swizzle follows the absolute shared address, so the shifted
      // views read the rows TMA wrote.  Descriptors of slot 0 are advanced by
      // the slot offsets (a descriptor's address field is the byte address
      // >> 4, and shared addresses stay below 256 KB, so adding never carries).
      constexpr uint32_t idesc = idesc_bf16_f32(128, 256, 1, 1);
      const uint64_t ad0 = sw128_desc(smem_u32(smem + kSOffKh), kSMnBlock, 1024);
      const uint64_t bd0 = sw128_desc(smem_u32(smem + kSOffV), 128, 1024);
      uint32_t hs = 0, hph = 0, os = 0, oph = 0;
      bool ok = true;
      for (long long r = blockIdx.x; r < R && ok; r += gridDim.x) {
        const long long se = range_begin(NS, R, r + 1);
        for (long long s = range_begin(NS, R, r); s < se && ok;) {
          const StageRef st = decode_stage(p, pre, s);
          const long long seg_end = min(se, st.s0 + st.nst);
          const int nst = (int)(seg_end - s);
          for (int it = 0; it < nst; ++it) {
            if (!mbar_wait(&kh_full[hs], hph, &ab) || !mbar_wait(&v_full[os], oph, &ab)) {
              if (!ab.raised()) report_error(4, ab);
              ok = false;
              break;
            }
            tc_fence_after();
            const uint64_t aoff = (uint64_t)(hs * kSKhStage) >> 4;
            const uint64_t boff = (uint64_t)(os * kSVStage) >> 4;
#pragma unroll
            for (int blk = 0; blk < 2; ++blk)
#pragma unroll
              for (int k16 = 0; k16 < kSTok / 16; ++k16)
                mma_bf16(tmem + 256 * blk, ad0 + aoff + (k16 * 2048 >> 4),
                         bd0 + boff + ((blk * kSVBlock + 16 * k16 * 128) >> 4), idesc,
                         (it | k16) != 0);
            mma_commit(&kh_empty[hs]);
            mma_commit(&v_empty[os]);
            if (++hs == kSKhStages) { hs = 0; hph ^= 1; }
            if (++os == kSVStages) { os = 0; oph ^= 1; }
          }
          if (ok) mma_commit(done);
          s = seg_end;
        }
      }
      mma_commit(fin);  // every MMA issued above has completed once this arrives
      if (!mbar_wait(fin, 0, nullptr)) report_error(8, ab);
    }
  }
  __syncthreads();
  if (warp == kSMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem, kSTmemCols);
  }
}

// Fixed-order combination of the partial records of one (b, h): the records
// q + r of the ranges r0..r1 meeting its sequence q, in range order,
//   M = max_j m_j,  S = sum_j e^{m_j - M} S_j / sum_j e^{m_j - M} l_j  (z likewise).
// Records go 32 at a time: lane j of every warp fetches record j's (m, l),
// the warp forms the batch maximum and the sum of l with shuffles (a fixed
// butterfly order), and each thread then accumulates its 4 state elements
// over the batch in record order, 16 loads in flight at a time, with the
// scale factors broadcast from the lanes that computed them.
//
// LEAN: 32 registers a thread, 4 loads in flight in registers and 5 more
// staged through shared memory by cp.async (10 KB).  The state kernel's 19
// warps leave exactly one 32-register warp per SM sub-partition free, and its
// shared memory leaves room for the staging buffer, so when the grid has at
// most one block per SM a lean block is made resident beside the state CTA as
// soon as the state grid signals its dependents, and waits there for the
// state grid to complete instead of being scheduled after it.  Lean blocks
// also serve grids too large for one wave of the wide ones (16 of them fit an
// SM, against a handful of wide blocks).
constexpr int kReduceThreads = 128;
template <int D, bool LEAN>
__global__ void __launch_bounds__(kReduceThreads, LEAN ? 16 : 1)
    tc_reduce_kernel(const float *__restrict__ records, const int32_t *__restrict__ seq_lens,
                     float *__restrict__ state, float2 *__restrict__ gate_stats, int B, int H,
                     int N, int P) {
  constexpr int G = kGroupCh / D;
  constexpr int REC = D * D + D + 4;
  constexpr int F = D * D + D;
  constexpr int CH = LEAN ? 4 : 16;   // record loads in flight per thread (registers)
  constexpr int SMR = LEAN ? 5 : 0;   // and staged through shared memory
  constexpr int CHT = CH + SMR;       // records per round trip
  __shared__ float4 stg[SMR > 0 ? SMR : 1][kReduceThreads];
  __shared__ int red[2][kReduceThreads / 32];
  // A lean block is resident while the state grid still runs: it lets the
  // readout launch only once the state is complete (below).  Other blocks
  // start after the state grid: the readout may be scheduled at once.
  if constexpr (!LEAN) grid_dep_launch();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int bh = blockIdx.x;
  const int b = bh / H, h = bh % H;
  const int hg = h / G, hh = h % G, HG = (H + G - 1) / G;
  const int e0 = (blockIdx.y * kReduceThreads + threadIdx.x) * 4;
  const bool act = e0 < F;  // every thread takes part in the shuffles
  const int L = clamp_len(seq_lens, b, N);
  const int nst = (L + kSTok - 1) / kSTok;
  // The record indices first: they depend only on the lengths (an input,
  // complete before the state kernel started), so this part runs while the
  // state kernel does.  NS stages in all, pre_b before batch row b (the state
  // kernel's stage prefix, formed here by the block).
  int NS, pre_b;
  if (seq_lens == nullptr) {
    NS = B * HG * nst;
    pre_b = b * HG * nst;
  } else {
    int sa = 0, sp = 0;
    for (int i = threadIdx.x; i < B; i += kReduceThreads) {
      const int c = HG * ((clamp_len(seq_lens, i, N) + kSTok - 1) / kSTok);
      sa += c;
      if (i < b) sp += c;
    }
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) {
      sa += __shfl_xor_sync(0xffffffffu, sa, o);
      sp += __shfl_xor_sync(0xffffffffu, sp, o);
    }
    if (lane == 0) {
      red[0][warp] = sa;
      red[1][warp] = sp;
    }
    __syncthreads();
    NS = pre_b = 0;
#pragma unroll
    for (int w = 0; w < kReduceThreads / 32; ++w) {
      NS += red[0][w];
      pre_b += red[1][w];
    }
  }
  long long r0 = 0;
  int nrec = 0, R = 1;
  if (nst > 0) {
    R = (NS + kRangeStages * P - 1) / (kRangeStages * P) * P;  // num_ranges
    const int s0 = pre_b + hg * nst;
    r0 = range_of(NS, R, s0);
    nrec = (int)(range_of(NS, R, s0 + nst - 1) - r0 + 1);
  }
  const bool may_be_empty = NS < R;  // otherwise every range holds a stage
  const float *rec0 = records + ((size_t)((long long)b * HG + hg + r0) * G + hh) * REC;
  const size_t rstride = (size_t)G * REC;
  const int ec = act ? e0 : 0;
  grid_dep_wait();  // the records come from the state kernel
  if constexpr (LEAN) grid_dep_launch();
  float M = -INFINITY, l = 0.f;
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  if (nst > 0) {
    const uint32_t stg0 = smem_u32(&stg[0][threadIdx.x]);
    for (int j0 = 0; j0 < nrec; j0 += 32) {
      const int nb = min(32, nrec - j0);
      // one round trip's loads (records k0 .. k0 + CHT - 1 of the batch; past
      // the batch the index is clamped to a record that exists): the first
      // SMR into this thread's shared-memory slots, the next CH into v
      float4 v[CH];
      auto issue = [&](int k0) {
        if constexpr (SMR > 0) {
#pragma unroll
          for (int k = 0; k < SMR; ++k) {
            const int kk = k0 + k < nb ? j0 + k0 + k : j0;
            cp_async_16(stg0 + (uint32_t)(k * kReduceThreads * 16),
                        rec0 + (size_t)kk * rstride + ec);
          }
          cp_async_commit();
        }
#pragma unroll
        for (int k = 0; k < CH; ++k) {
          const int kk = k0 + SMR + k < nb ? j0 + k0 + SMR + k : j0;
          v[k] = __ldg((const float4 *)(rec0 + (size_t)kk * rstride + ec));
        }
      };
      // the first loads go out with the (m, l) loads: they do not depend on
      // the scale factors
      issue(0);
      const int j = j0 + lane;
      bool has = j < nrec;
      if (has && may_be_empty)  // with fewer stages than ranges some left no record
        has = range_begin(NS, R, r0 + j) < range_begin(NS, R, r0 + j + 1);
      const float *rj = rec0 + (size_t)j * rstride;
      const float mj = has ? __ldg(rj + F) : -INFINITY;
      const float lj = has ? __ldg(rj + F + 1) : 0.f;
      float Mb = mj;
#pragma unroll
      for (int o = 16; o >= 1; o >>= 1) Mb = fmaxf(Mb, __shfl_xor_sync(0xffffffffu, Mb, o));
      if (Mb > M) {  // rescale the running sums to the new maximum
        const float rsc = (M == -INFINITY) ? 0.f : __expf(M - Mb);
        acc.x *= rsc; acc.y *= rsc; acc.z *= rsc; acc.w *= rsc;
        l *= rsc;
        M = Mb;
      }
      const float sc = has ? __expf(mj - M) : 0.f;
      float ls = sc * lj;
#pragma unroll
      for (int o = 16; o >= 1; o >>= 1) ls += __shfl_xor_sync(0xffffffffu, ls, o);
      l += ls;
      auto fma4 = [&](float s4, const float4 &x) {
        acc.x = fmaf(s4, x.x, acc.x);
        acc.y = fmaf(s4, x.y, acc.y);
        acc.z = fmaf(s4, x.z, acc.z);
        acc.w = fmaf(s4, x.w, acc.w);
      };
      for (int k0 = 0; k0 < nb; k0 += CHT) {
        if (k0 > 0) issue(k0);
        // in record order; a zero factor marks a record that does not exist
        // (an empty range, whose slot holds whatever was there) or that
        // underflowed: skip it
        if constexpr (SMR > 0) {
          cp_async_wait_all();  // this thread's own copies: no barrier needed
#pragma unroll
          for (int k = 0; k < SMR; ++k) {
            const float skk = __shfl_sync(0xffffffffu, sc, (k0 + k) & 31);
            if (k0 + k < nb && skk != 0.f) fma4(skk, stg[k][threadIdx.x]);
          }
        }
#pragma unroll
        for (int k = 0; k < CH; ++k) {
          const float skk = __shfl_sync(0xffffffffu, sc, (k0 + SMR + k) & 31);
          if (k0 + SMR + k < nb && skk != 0.f) fma4(skk, v[k]);
        }
      }
    }
  }
  if (gate_stats != nullptr && blockIdx.y == 0 && threadIdx.x == 0)
    gate_stats[bh] = make_float2(M, l);  // every thread of bh holds the same pair
  if (!act) return;
  const float inv = l > 0.f ? 1.f / l : 0.f;
  // record position e0 of S ([c / 8][a][c % 8]) -> state element a D + c
  const int se = e0 < D * D ? (e0 % (D * 8)) / 8 * D + e0 / (D * 8) * 8 + e0 % 8 : e0;
  *(float4 *)(state + (size_t)bh * F + se) =
      make_float4(acc.x * inv, acc.y * inv, acc.z * inv, acc.w * inv);
}

// ===================================================================== readout
struct ReadoutParams {
  const __nv_bfloat16 *q;
  const float *conv_w, *norm_w, *state;
  const int32_t *seq_lens;
  __nv_bfloat16 *o;
  float *o32;      // fp32 output of the debug instantiation (F32O), else unused
  int B, H, N;
  float eps;
  int wait_late;   // only the reads of `state` wait for the preceding kernel
  uint32_t flags;  // gbla_flags (NO_CONV, NO_NORM)
};

// phi(conv(q)) for 4 consecutive rows of one producer sub-stream; xm holds the
// window before the first row; rows are read by `row_raw(u)` (u = 0..3).
template <typename RowFn>
__device__ __forceinline__ void readout_rows4(const float (&wq)[4][8], float (&xm)[3][8],
                                              RowFn row_raw, uint32_t abase,
                                              const uint32_t *aoff) {
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    float x[8];
    unpack8(row_raw(u), x);
    uint32_t pq[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 ph = phi2_log2(conv2(wq, xm, x, 2 * i));
      pq[i] = f2_to_bf2(ph.x, ph.y);
    }
    slide(xm, x);
    sts_v4(abase + aoff[u], make_uint4(pq[0], pq[1], pq[2], pq[3]));
  }
}

// Position in the flattened (batch, head, 128-token tile) order of the readout.
struct TileCursor {
  int b, h, r0, nrow, L;
};
__device__ __forceinline__ TileCursor tile_at(const int *pre, const int32_t *seq_lens, int B,
                                              int N, int i) {
  TileCursor t;
  t.b = find_batch(pre, B, i);
  t.L = clamp_len(seq_lens, t.b, N);
  const int nt = (t.L + kRTok - 1) / kRTok;
  const int r = i - pre[t.b];
  t.h = r / nt;
  t.r0 = (r % nt) * kRTok;
  t.nrow = min(kRTok, t.L - t.r0);
  return t;
}
// The next tile; only called while one remains.
__device__ __forceinline__ void tile_next(TileCursor &t, const int32_t *seq_lens, int B, int H,
                                          int N) {
  t.r0 += kRTok;
  if (t.r0 >= t.L) {
    t.r0 = 0;
    if (++t.h == H) {
      t.h = 0;
      do {
        ++t.b;
        t.L = t.b < B ? clamp_len(seq_lens, t.b, N) : 0;
      } while (t.b < B && t.L == 0);
    }
  }
  t.nrow = min(kRTok, t.L - t.r0);
}

// F32O: the debug instantiation behind gbla_forward_f32out.  It runs the same
// arithmetic and stores each y in fp32 (plain stores of the valid rows) where
// the product instantiation rounds it to bf16 and stores the tile with TMA.
template <int D, bool ABL, bool F32O>
__global__ void __launch_bounds__(kRThreads, 1)
    tc_readout_kernel(const ReadoutParams p, const __grid_constant__ CUtensorMap tm_og,
                      const __grid_constant__ CUtensorMap tm_o,
                      const __grid_constant__ CUtensorMap tm_q) {
  using C = ReadoutCfg<D>;
  constexpr int NR = C::NR;
  constexpr int OGS = C::kOgStages;
  constexpr int QS = C::kQStages > 0 ? C::kQStages : 1;
  constexpr int F = D * D + D;
  constexpr int CPE = D / 2;  // columns per epilogue warp
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  int *pre = (int *)(smem + C::kOffPre);
  uint64_t *bars = (uint64_t *)(smem + C::kOffBar);
  uint64_t *a_full = bars, *a_empty = bars + 2, *og_full = bars + 4, *og_empty = og_full + OGS,
           *q_full = og_empty + OGS, *q_empty = q_full + C::kQStages,
           *acc_full = q_empty + C::kQStages, *acc_empty = acc_full + 2,
           *b_full = acc_empty + 2, *b_free = b_full + 1, *fin = b_free + 1;
  uint32_t *tmem_slot = (uint32_t *)(smem + C::kOffMisc);
  const AbortFlag ab{smem_u32(smem + C::kOffMisc + 4)};
  __shared__ int s_tot[8];

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int B = p.B, H = p.H, N = p.N;
  const uint32_t flags = ABL ? p.flags : 0u;  // ablations (see tc_state_kernel)

  if (tid == 0) {
    *(volatile int *)(smem + C::kOffMisc + 4) = 0;
    for (int i = 0; i < 2; ++i) {
      mbar_init(&a_full[i], kRProdWarps);
      mbar_init(&a_empty[i], 1);
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], kREpiWarps);
    }
    for (int i = 0; i < OGS; ++i) {
      mbar_init(&og_full[i], 1);
      mbar_init(&og_empty[i], kREpiWarps / 2);  // one release per TMEM lane quarter
    }
    for (int i = 0; i < C::kQStages; ++i) {
      mbar_init(&q_full[i], 1);
      mbar_init(&q_empty[i], kRProdWarps);
    }
    mbar_init(b_full, kREpiWarps);
    mbar_init(b_free, 1);
    mbar_init(fin, 1);
    fence_mbar_init();
  }
  if (warp == kRTmaWarp && lane == 0) {
    tma_prefetch_desc(&tm_og);
    tma_prefetch_desc(&tm_o);
    tma_prefetch_desc(&tm_q);
  }
  // Everything below may read what earlier work on the stream wrote, unless
  // that work is the state reduction, which only `state` depends on.
  if (!p.wait_late) grid_dep_wait();
  // The next kernel on the stream may launch now: its CTAs take the SMs as
  // these leave.  A dependent that reads what this grid writes waits for it
  // to complete (the state kernel does so before its first read).
  grid_dep_launch();
  if (warp < 4) {
    prefix_counts(pre, B, tid, 128, 1, s_tot, [&](int b) {
      const int L = clamp_len(p.seq_lens, b, N);
      return H * ((L + kRTok - 1) / kRTok);
    });
  }
  __syncthreads();
  const int T = pre[B];
  const long long i0 = (long long)T * blockIdx.x / gridDim.x;
  const long long i1 = (long long)T * (blockIdx.x + 1) / gridDim.x;
  if (i0 >= i1) return;
  if (warp == kRMmaWarp) tmem_alloc(tmem_slot, C::kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  // Tile -> (b, h, first token, valid rows): decoded once, then stepped; each
  // role calls tile_of for ii = i0, i0 + 1, ... in order.
  TileCursor tc0 = tile_at(pre, p.seq_lens, B, N, (int)i0);
  auto tile_of = [&](long long ii, int &b, int &h, int &r0, int &nrow) {
    if (ii != i0) tile_next(tc0, p.seq_lens, B, H, N);
    b = tc0.b;
    h = tc0.h;
    r0 = tc0.r0;
    nrow = tc0.nrow;
  };

  if (warp < kRProdWarps) {
    // ------------------------------------------------------------ producers: phi(conv(q))
    constexpr int TPR = C::TPR, TPS = C::TPS, NCH = C::NCH;
    const int c = tid % TPR, stream = tid / TPR;
    const int kb = (NCH * c) >> 6, cc = ((NCH * c) & 63) >> 3;  // 64-channel block, 16-byte chunk
    const int row0 = stream * TPS;  // first tile row of this sub-stream
    // swizzled offsets of this thread's 16-byte pieces of A rows row0 + u
    // (the TMA q path uses one 8-row atom per sub-stream and needs none)
    // (QA: offsets of the slot rows row0 + 3 + u, which hold the raw q of this
    // sub-stream's tokens and receive A rows row0 + u in place)
    uint32_t aoff[C::QT ? 1 : TPS];
    if constexpr (!C::QT) {
#pragma unroll
      for (int u = 0; u < TPS; ++u) {
        const int row = row0 + u + (C::QA ? 3 : 0);
        aoff[u] = kb * C::kABlk + (row >> 3) * 1024 + (row & 7) * 128 + ((cc ^ (row & 7)) << 4);
      }
    }
    // TMA q path: q tile row j holds token r0 - 3 + j; this thread reads rows
    // row0 + k (k = 0..10, 4 channels = 8 bytes) and writes A rows row0 + u
    const uint32_t thr8 = (uint32_t)(stream * 1024 + (c & 1) * 8);
    int cur_b = -1, cur_h = -1;
    float wq[4][NCH];
    for (long long ii = i0; ii < i1; ++ii) {
      int b, h, r0, nrow;
      tile_of(ii, b, h, r0, nrow);
      const int li = (int)(ii - i0);
      if (b != cur_b || h != cur_h) {
        // New (b, h): the q taps, pre-scaled by log2(e) (phi2_log2 takes
        // x log2(e)); 4 NCH consecutive floats per thread.  B = [S | z] is
        // rebuilt by the epilogue warps.
#pragma unroll
        for (int i = 0; i < NCH; ++i) {
          const float4 t4 = (flags & GBLA_FLAG_NO_CONV)
                                ? make_float4(0.f, 0.f, 0.f, 1.f)  // identity taps (ablation)
                                : __ldg((const float4 *)(p.conv_w + ((size_t)h * D + NCH * c + i) * 4));
          wq[0][i] = t4.x * kLog2e;
          wq[1][i] = t4.y * kLog2e;
          wq[2][i] = t4.z * kLog2e;
          wq[3][i] = t4.w * kLog2e;
        }
        cur_b = b;
        cur_h = h;
      }
      const int sa = li & 1;
      if constexpr (C::QA) {  // the raw q tile has landed in the slot (freed by the MMA before)
        if (!mbar_wait(&q_full[sa], (li >> 1) & 1, &ab) && !ab.raised()) report_error(32, ab);
      } else {
        if (!mbar_wait(&a_empty[sa], ((li >> 1) & 1) ^ 1, &ab) && !ab.raised())
          report_error(32, ab);
      }
      const uint32_t abase = smem_u32(smem + C::kOffA + sa * C::kABytes);
      if constexpr (C::QA) {
        // slot row j holds token r0 - 3 + j; this thread reads rows row0 .. row0
        // + 10 of its 8 channels and rewrites rows row0 + 3 .. row0 + 10 (A rows
        // row0 .. row0 + 7).  The 3 history rows are read before the producers'
        // barrier, since the sub-stream before rewrites them; each other row is
        // read by its own thread just before it rewrites it.
        float xm[3][8];
#pragma unroll
        for (int u = 0; u < 3; ++u) {
          const int row = row0 + u;
          unpack8(lds_v4(abase + kb * C::kABlk + row * 128 + ((cc ^ (row & 7)) << 4)), xm[u]);
        }
        named_barrier(2, kRProd);
#pragma unroll
        for (int g4 = 0; g4 < TPS; g4 += 4)
          readout_rows4(wq, xm, [&](int u) { return lds_v4(abase + aoff[g4 + u]); }, abase,
                        aoff + g4);
      } else if constexpr (C::QT) {
        // q tile from TMA (128-byte swizzle); rows row0 .. row0 + 10 hold this
        // sub-stream's 3 history tokens and its 8 tokens
        const int sq = li % QS;
        if (!mbar_wait(&q_full[sq], (li / QS) & 1, &ab) && !ab.raised()) report_error(32, ab);
        const uint32_t qb = smem_u32(smem + C::kOffQ + sq * C::kQBytes) + thr8;
        float x[TPS + 3][4];
#pragma unroll
        for (int k = 0; k < TPS + 3; ++k)
          unpack4(lds_v2(qb + (k >> 3) * 1024 + (k & 7) * 128 + ((cc ^ (k & 7)) << 4)), x[k]);
        __syncwarp();
        if (lane == 0) mbar_arrive(&q_empty[sq]);
        const uint32_t at = abase + thr8;
#pragma unroll
        for (int u = 0; u < TPS; ++u) {
          const float2 p01 = phi2_log2(conv_rows_n(wq, x, u, 0));
          const float2 p23 = phi2_log2(conv_rows_n(wq, x, u, 2));
          sts_v2(at + u * 128 + ((cc ^ u) << 4), f2_to_bf2(p01.x, p01.y), f2_to_bf2(p23.x, p23.y));
        }
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&a_full[sa]);
    }
  } else if (warp < kRMmaWarp) {
    // ------------------------------------------------------------ epilogue
    const int ew = warp - kRProdWarps;           // 0..7
    const int q4 = ew & 3, part = ew >> 2;       // TMEM lane quarter, column half
    const int row = 32 * q4 + lane;
    const uint32_t ss_s = smem_u32(smem + C::kOffSs);
    constexpr int NH = CPE / 32;                 // 32-column pieces per warp
    // swizzled offsets of this row's 8-channel pieces in an out_gate/o tile
    uint32_t ogoff[CPE / 8];
#pragma unroll
    for (int g8 = 0; g8 < CPE / 8; ++g8) {
      const int ch0 = part * CPE + 8 * g8;
      const int kbo = ch0 >> 6, cco = (ch0 & 63) >> 3;
      ogoff[g8] = kbo * (kRTok * 128) + (row >> 3) * 1024 + (row & 7) * 128 + ((cco ^ (row & 7)) << 4);
    }
    int pend = -1;  // og stage whose TMA store may still be reading it (leader only)
    // B = [S | z | 0] of (b, h) as bf16 hi/lo, K-major, 128B swizzle, rebuilt
    // for the first tile and before the first tile of every new (b, h), once
    // the MMAs that read the previous one have completed (b_free).
    int nbh = 0;
    const int etid = tid - kRProd;
    auto build_b = [&](int b, int h) {
      if (nbh > 0 && !mbar_wait(b_free, (nbh - 1) & 1, &ab) && !ab.raised()) report_error(16, ab);
      if (nbh == 0) grid_dep_wait();  // the state comes from the preceding kernel
      const float *st = p.state + ((size_t)b * H + h) * F;
      constexpr int NI = NR * (D / 8);  // (row e of B, 8-element K chunk ck) items
      constexpr int BU = (NI + kREpi - 1) / kREpi < 3 ? (NI + kREpi - 1) / kREpi : 3;
      for (int item0 = etid; item0 < NI; item0 += BU * kREpi) {
        float vals[BU][8];  // all items' loads in flight together
#pragma unroll
        for (int u = 0; u < BU; ++u) {
          const int item = item0 + u * kREpi;
          const int e = item % NR, ck = item / NR;
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const int d = 8 * ck + i;
            vals[u][i] = item < NI && e < D ? st[(size_t)d * D + e]
                                            : (item < NI && e == D ? st[D * D + d] : 0.f);
          }
        }
#pragma unroll
        for (int u = 0; u < BU; ++u) {
          const int item = item0 + u * kREpi;
          if (item >= NI) break;
          const int e = item % NR, ck = item / NR;
          uint32_t hi[4], lo[4];
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            hi[i] = f2_to_bf2(vals[u][2 * i], vals[u][2 * i + 1]);
            const float2 r2 = __ffma2_rn(bf2_to_f2(hi[i]), make_float2(-1.f, -1.f),
                                         make_float2(vals[u][2 * i], vals[u][2 * i + 1]));
            lo[i] = f2_to_bf2(r2.x, r2.y);
          }
          const int kbk = ck >> 3, ckk = ck & 7;
          const uint32_t off = kbk * (NR * 128) + (e >> 3) * 1024 + (e & 7) * 128 +
                               ((ckk ^ (e & 7)) << 4);
          sts_v4(smem_u32(smem + C::kOffBhi) + off, make_uint4(hi[0], hi[1], hi[2], hi[3]));
          sts_v4(smem_u32(smem + C::kOffBlo) + off, make_uint4(lo[0], lo[1], lo[2], lo[3]));
        }
      }
      // the head's norm weights for the epilogue, read back after barrier 7
      if (etid < D / 4)
        *(float4 *)(smem + C::kOffW + 16 * etid) = __ldg((const float4 *)(p.norm_w + (size_t)h * D) + etid);
      fence_proxy_async_smem();
      named_barrier(7, kREpi);
      if (lane == 0) mbar_arrive(b_full);
      ++nbh;
    };
    build_b(tc0.b, tc0.h);
    for (long long ii = i0; ii < i1; ++ii) {
      int b, h, r0, nrow;
      tile_of(ii, b, h, r0, nrow);
      const int li = (int)(ii - i0);
      const int abuf = li & 1, so = li % OGS;
      if (!mbar_wait(&acc_full[abuf], (li >> 1) & 1, &ab) && !ab.raised()) report_error(64, ab);
      if (!mbar_wait(&og_full[so], (li / OGS) & 1, &ab) && !ab.raised()) report_error(64, ab);
      tc_fence_after();
      const uint32_t tacc = tmem + ((uint32_t)(32 * q4) << 16) + abuf * C::kAccStride;
      const uint32_t tcol = tacc + part * CPE;
      // pass 1: this warp's half-row sum of squares of the numerators
      float den[8], va[16], vb[16];
      float2 ss2 = make_float2(0.f, 0.f);
#pragma unroll
      for (int h2 = 0; h2 < NH; ++h2) {
        if (h2 == 0) tmem_ld8(tacc + D, den);
        tmem_ld16(tcol + 32 * h2, va);
        tmem_ld16(tcol + 32 * h2 + 16, vb);
        tmem_ld_wait_regs(va);
        tmem_ld_wait_regs(vb);
        if (h2 == 0) tmem_ld_wait_regs(den);
#pragma unroll
        for (int i = 0; i < 16; i += 2) {
          ss2 = __ffma2_rn(make_float2(va[i], va[i + 1]), make_float2(va[i], va[i + 1]), ss2);
          ss2 = __ffma2_rn(make_float2(vb[i], vb[i + 1]), make_float2(vb[i], vb[i + 1]), ss2);
        }
      }
      // the two warps of a lane quarter exchange their half-row sums of squares
      sts_f32(ss_s + (uint32_t)(part * 128 + row) * 4, ss2.x + ss2.y);
      named_barrier(3 + q4, 64);
      const float ss = lds_f32(ss_s + (uint32_t)row * 4) + lds_f32(ss_s + (uint32_t)(128 + row) * 4);
      // O = acc / den;  y = O / sqrt(mean O^2 + eps) * w * silu(og) = acc * rr * w * silu(og)
      const float inv = rcp_approx(den[0]);
      const float ms = ss * inv * inv * (1.f / (float)D);
      const float rr = rsqrtf(ms + p.eps) * inv;
      const bool no_norm = flags & GBLA_FLAG_NO_NORM;
      const uint32_t nws = smem_u32(smem + C::kOffW) + (uint32_t)(part * CPE) * 4;
      const uint32_t ogt = smem_u32(smem + C::kOffOg + so * C::kOgBytes);
      auto og_addr = [&](int col) {  // col: channel offset within this warp's half
        return ogt + ogoff[col / 8];
      };
#pragma unroll
      for (int h2 = 0; h2 < NH; ++h2) {
        if (NH > 1) {  // pass 1 kept only the last piece in registers
          tmem_ld16(tcol + 32 * h2, va);
          tmem_ld16(tcol + 32 * h2 + 16, vb);
          tmem_ld_wait_regs(va);
          tmem_ld_wait_regs(vb);
        }
        // four groups of 8 channels; out_gate and weights of the next group in flight
        uint4 gcur = lds_v4(og_addr(32 * h2));
        uint4 wr0 = lds_v4(nws + (32 * h2) * 4), wr1 = lds_v4(nws + (32 * h2 + 4) * 4);
        float4 wc0 = make_float4(__uint_as_float(wr0.x), __uint_as_float(wr0.y),
                                 __uint_as_float(wr0.z), __uint_as_float(wr0.w));
        float4 wc1 = make_float4(__uint_as_float(wr1.x), __uint_as_float(wr1.y),
                                 __uint_as_float(wr1.z), __uint_as_float(wr1.w));
#pragma unroll
        for (int g = 0; g < 4; ++g) {
          uint4 gnext = gcur;
          float4 wn0 = wc0, wn1 = wc1;
          if (g < 3) {
            gnext = lds_v4(og_addr(32 * h2 + 8 * (g + 1)));
            const uint4 r0 = lds_v4(nws + (32 * h2 + 8 * (g + 1)) * 4);
            const uint4 r1 = lds_v4(nws + (32 * h2 + 8 * (g + 1) + 4) * 4);
            wn0 = make_float4(__uint_as_float(r0.x), __uint_as_float(r0.y), __uint_as_float(r0.z),
                              __uint_as_float(r0.w));
            wn1 = make_float4(__uint_as_float(r1.x), __uint_as_float(r1.y), __uint_as_float(r1.z),
                              __uint_as_float(r1.w));
          }
          float gv[8];
          unpack8(gcur, gv);
          const float wv8[8] = {wc0.x, wc0.y, wc0.z, wc0.w, wc1.x, wc1.y, wc1.z, wc1.w};
          const float *acc8 = g < 2 ? &va[8 * g] : &vb[8 * (g - 2)];
          float2 y[4];
          if (no_norm) {  // ablation without the gated RMSNorm: o = O = acc / den
#pragma unroll
            for (int i = 0; i < 4; ++i)
              y[i] = __fmul2_rn(make_float2(acc8[2 * i], acc8[2 * i + 1]), make_float2(inv, inv));
          } else {
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              // silu(g) = g sigmoid(g) = h + h tanh(h),  h = g / 2
              const float2 hg = __fmul2_rn(make_float2(gv[2 * i], gv[2 * i + 1]),
                                           make_float2(0.5f, 0.5f));
              const float2 sg =
                  __ffma2_rn(hg, make_float2(tanh_approx(hg.x), tanh_approx(hg.y)), hg);
              const float2 av = __fmul2_rn(make_float2(acc8[2 * i], acc8[2 * i + 1]),
                                           make_float2(wv8[2 * i], wv8[2 * i + 1]));
              y[i] = __fmul2_rn(__fmul2_rn(av, sg), make_float2(rr, rr));
            }
          }
          if constexpr (F32O) {
            if (row < nrow) {
              float4 *dst = (float4 *)(p.o32 + (((size_t)b * N + r0 + row) * H + h) * D +
                                       part * CPE + 32 * h2 + 8 * g);
              dst[0] = make_float4(y[0].x, y[0].y, y[1].x, y[1].y);
              dst[1] = make_float4(y[2].x, y[2].y, y[3].x, y[3].y);
            }
          } else {
            sts_v4(og_addr(32 * h2 + 8 * g),
                   make_uint4(f2_to_bf2(y[0].x, y[0].y), f2_to_bf2(y[1].x, y[1].y),
                              f2_to_bf2(y[2].x, y[2].y), f2_to_bf2(y[3].x, y[3].y)));
          }
          gcur = gnext;
          wc0 = wn0;
          wc1 = wn1;
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acc_empty[abuf]);
      // Each lane quarter's 32 rows (both halves) go out on their own: the
      // pair meets on its named barrier, then one thread stores them with TMA
      // (full tiles) or releases the buffer after the direct stores (tail).
      const bool leader = part == 0 && lane == 0;
      if (!F32O && nrow == kRTok) {
        fence_proxy_async_smem();
        named_barrier(3 + q4, 64);
        if (leader) {
#pragma unroll
          for (int kbo = 0; kbo < C::KB; ++kbo)
            tma_store_4d(&tm_o, smem + C::kOffOg + so * C::kOgBytes + kbo * (kRTok * 128) +
                                    q4 * (32 * 128),
                         kbo * 64, h, r0 + 32 * q4, b);
          tma_store_commit();
          if constexpr (OGS >= 3) {
            // release the previous tile's buffer once its store has read it; this
            // tile's buffer is released one tile later, so the store overlaps work
            if (pend >= 0) {
              tma_store_wait_read<1>();
              mbar_arrive(&og_empty[pend]);
            }
            pend = so;
          } else {
            tma_store_wait_read<0>();
            mbar_arrive(&og_empty[so]);
          }
        }
        __syncwarp();
      } else {
        // Ragged tail: rows past the sequence end must not be written (the
        // fp32 debug output was stored above).
        if (!F32O && row < nrow) {
          __nv_bfloat16 *orow = p.o + (((size_t)b * N + r0 + row) * H + h) * D + part * CPE;
#pragma unroll
          for (int cb = 0; cb < CPE; cb += 8) *(uint4 *)(orow + cb) = lds_v4(og_addr(cb));
        }
        named_barrier(3 + q4, 64);
        if (leader) {
          if (pend >= 0) {
            tma_store_wait_read<0>();
            mbar_arrive(&og_empty[pend]);
            pend = -1;
          }
          mbar_arrive(&og_empty[so]);
        }
        __syncwarp();
      }
      if (ii + 1 < i1) {  // the next tile starts a new (b, h): its B, once this one's MMAs are done
        TileCursor nx = tc0;
        tile_next(nx, p.seq_lens, B, H, N);
        if (nx.b != b || nx.h != h) build_b(nx.b, nx.h);
      }
    }
    if (part == 0 && lane == 0) tma_store_wait_all<0>();
  } else if (warp == kRMmaWarp) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      int cur_b = -1, cur_h = -1, nbh = 0;
      for (long long ii = i0; ii < i1; ++ii) {
        int b, h, r0, nrow;
        tile_of(ii, b, h, r0, nrow);
        const int li = (int)(ii - i0);
        bool ok = true;
        if (b != cur_b || h != cur_h) {
          ok = mbar_wait(b_full, nbh & 1, &ab);
          cur_b = b;
          cur_h = h;
          ++nbh;
        }
        const int sa = li & 1, abuf = li & 1;
        ok = ok && mbar_wait(&a_full[sa], (li >> 1) & 1, &ab) &&
             mbar_wait(&acc_empty[abuf], ((li >> 1) & 1) ^ 1, &ab);
        if (!ok) {
          if (!ab.raised()) report_error(128, ab);
          break;
        }
        tc_fence_after();
        const uint32_t abase = smem_u32(smem + C::kOffA + sa * C::kABytes);
        const uint32_t bhi = smem_u32(smem + C::kOffBhi), blo = smem_u32(smem + C::kOffBlo);
        const uint32_t dacc = tmem + abuf * C::kAccStride;
#pragma unroll
        for (int kbk = 0; kbk < C::KB; ++kbk)
#pragma unroll
          for (int k16 = 0; k16 < 4; ++k16) {
            const uint32_t ao = kbk * C::kABlk + C::kARow0 + k16 * 32;
            const uint32_t bo = kbk * (NR * 128) + k16 * 32;
            const uint64_t ad = sw128_desc(abase + ao, 16, 1024);
            mma_bf16(dacc, ad, sw128_desc(bhi + bo, 16, 1024), C::kIdesc, (kbk | k16) != 0);
            mma_bf16(dacc, ad, sw128_desc(blo + bo, 16, 1024), C::kIdesc, 1);
          }
        mma_commit(&a_empty[sa]);
        mma_commit(&acc_full[abuf]);
        // last tile of this (b, h) in this CTA: release B for the next rebuild
        bool last = ii + 1 >= i1;
        if (!last) {
          TileCursor nx = tc0;
          tile_next(nx, p.seq_lens, B, H, N);
          last = (nx.b != b || nx.h != h);
        }
        if (last) mma_commit(b_free);
      }
      mma_commit(fin);  // every MMA issued above has completed once this arrives
      if (!mbar_wait(fin, 0, nullptr)) report_error(256, ab);
    }
  } else if (warp == kRTmaWarp) {
    // ------------------------------------------------------------ TMA: out_gate
    if (lane == 0) {
      const uint64_t pol = l2_policy_evict_first();  // read once
      for (long long ii = i0; ii < i1; ++ii) {
        int b, h, r0, nrow;
        tile_of(ii, b, h, r0, nrow);
        const int li = (int)(ii - i0);
        const int so = li % OGS;
        if (!mbar_wait(&og_empty[so], ((li / OGS) & 1) ^ 1, &ab)) {
          if (!ab.raised()) report_error(512, ab);
          break;
        }
        uint8_t *dst = smem + C::kOffOg + so * C::kOgBytes;
        mbar_arrive_expect_tx(&og_full[so], C::kOgBytes);
#pragma unroll
        for (int kbo = 0; kbo < C::KB; ++kbo)
          tma_load_4d_hint(dst + kbo * (kRTok * 128), &tm_og, &og_full[so], kbo * 64, h, r0, b,
                           pol);
      }
    }
  } else {
    // ------------------------------------------------------------ TMA: q
    if (lane == 0 && C::QA) {  // into the A slot, once the MMA has read it
      const uint64_t pol = l2_policy_evict_first();
      for (long long ii = i0; ii < i1; ++ii) {
        int b, h, r0, nrow;
        tile_of(ii, b, h, r0, nrow);
        const int li = (int)(ii - i0), sa = li & 1;
        if (!mbar_wait(&a_empty[sa], ((li >> 1) & 1) ^ 1, &ab)) {
          if (!ab.raised()) report_error(1024, ab);
          break;
        }
        mbar_arrive_expect_tx(&q_full[sa], C::KB * C::kQTileBytes);
#pragma unroll
        for (int kbo = 0; kbo < C::KB; ++kbo)
          tma_load_4d_hint(smem + C::kOffA + sa * C::kABytes + kbo * C::kABlk, &tm_q, &q_full[sa],
                           kbo * 64, h, r0 - 3, b, pol);
      }
    }
    if (lane == 0 && C::QT) {
      const uint64_t pol = l2_policy_evict_first();  // read once (3 halo rows aside)
      for (long long ii = i0; ii < i1; ++ii) {
        int b, h, r0, nrow;
        tile_of(ii, b, h, r0, nrow);
        const int li = (int)(ii - i0);
        const int sq = li % QS;
        if (!mbar_wait(&q_empty[sq], ((li / QS) & 1) ^ 1, &ab)) {
          if (!ab.raised()) report_error(1024, ab);
          break;
        }
        mbar_arrive_expect_tx(&q_full[sq], C::kQTileBytes);
        tma_load_4d_hint(smem + C::kOffQ + sq * C::kQBytes, &tm_q, &q_full[sq], 0, h, r0 - 3, b,
                         pol);
      }
    }
  }
  __syncthreads();
  if (warp == kRMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem, C::kTmemCols);
  }
}

// ===================================================================== host side
using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                   const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                   const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = (EncodeTiledFn)f;
  });
  return fn;
}

// 4-D map over a [B, N, H, D] bf16 tensor; box = 64 channels x 1 head x `rows`
// tokens, 128-byte swizzle (the layout the readout's producers and epilogue read).
cudaError_t make_bnhd_map(CUtensorMap *m, const void *base, int B, int N, int H, int D,
                          int rows) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return cudaErrorNotSupported;
  const cuuint64_t dims[4] = {(cuuint64_t)D, (cuuint64_t)H, (cuuint64_t)N, (cuuint64_t)B};
  const cuuint64_t strides[3] = {(cuuint64_t)D * 2, (cuuint64_t)H * D * 2,
                                 (cuuint64_t)N * H * D * 2};
  const cuuint32_t box[4] = {64, 1, (cuuint32_t)rows, 1};
  const cuuint32_t estr[4] = {1, 1, 1, 1};
  // A token's row of one head is D * 2 bytes; promoting a 128-byte row to a
  // 256-byte L2 fill would also fetch the neighbouring head, which another CTA
  // reads much later, so D = 64 rows are fetched at their own size.
  const CUtensorMapL2promotion promo =
      D * 2 >= 256 ? CU_TENSOR_MAP_L2_PROMOTION_L2_256B : CU_TENSOR_MAP_L2_PROMOTION_L2_128B;
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(base), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, promo,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

// 4-D map over a [B, N, H, D] bf16 tensor for the state kernel's raw tiles:
// box = one head group (128 channels) x kSRawRows tokens, no swizzle, so a
// token's group row is 256 contiguous bytes in shared memory.
cudaError_t make_group_map(CUtensorMap *m, const void *base, int B, int N, int H, int D) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return cudaErrorNotSupported;
  const cuuint64_t dims[4] = {(cuuint64_t)D, (cuuint64_t)H, (cuuint64_t)N, (cuuint64_t)B};
  const cuuint64_t strides[3] = {(cuuint64_t)D * 2, (cuuint64_t)H * D * 2,
                                 (cuuint64_t)N * H * D * 2};
  const cuuint32_t box[4] = {(cuuint32_t)D, (cuuint32_t)(kGroupCh / D), (cuuint32_t)kSRawRows, 1};
  const cuuint32_t estr[4] = {1, 1, 1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(base), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

struct DeviceInfo {
  int sms = 0;
  bool sm103 = false;
};
constexpr int kMaxDevices = 128;
DeviceInfo g_dev_info[kMaxDevices];
std::once_flag g_dev_once[kMaxDevices];

const DeviceInfo &device_info() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) dev = 0;
  std::call_once(g_dev_once[dev], [dev] {
    int n = 0, major = 0, minor = 0;
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
    g_dev_info[dev].sms = n > 0 ? n : 1;
    g_dev_info[dev].sm103 = (major == 10 && minor == 3);
  });
  return g_dev_info[dev];
}

int num_sms() { return device_info().sms; }

// Partial records the state step may write: one per (sequence, range) meeting,
// at most R + Q - 1 with R bounded by the stage count of full-length sequences.
size_t record_slots(const Problem &p) {
  const int G = kGroupCh / p.D;
  const long long Q = (long long)p.B * ((p.H + G - 1) / G);
  const long long ns_max = Q * ((p.N + kSTok - 1) / kSTok);
  return (size_t)(num_ranges(ns_max, num_sms()) + Q);
}
size_t records_bytes(const Problem &p) {
  const int G = kGroupCh / p.D;
  return record_slots(p) * G * ((size_t)p.D * p.D + p.D + 4) * sizeof(float);
}

template <int D>
cudaError_t run_state(const Problem &p, const void *k, const void *v, const void *gate,
                      const float *conv_w, void *ws, float *state, cudaStream_t st,
                      float2 *gate_stats) {
  constexpr int G = kGroupCh / D;
  StateParams sp;
  sp.gate = (const __nv_bfloat16 *)gate;
  sp.conv_w = conv_w;
  sp.seq_lens = p.seq_lens;
  sp.records = (float *)ws;
  sp.B = p.B;
  sp.H = p.H;
  sp.N = p.N;
  sp.flags = p.flags;
  sp.HG = (p.H + G - 1) / G;
  CUtensorMap tm_k, tm_v;
  cudaError_t e = make_group_map(&tm_k, k, p.B, p.N, p.H, D);
  if (e != cudaSuccess) return e;
  if ((e = make_bnhd_map(&tm_v, v, p.B, p.N, p.H, D, kSRawRows)) != cudaSuccess) return e;
  auto k1 = p.flags ? tc_state_kernel<D, true> : tc_state_kernel<D, false>;
  if ((e = cudaFuncSetAttribute(k1, cudaFuncAttributeMaxDynamicSharedMemorySize, kSSmemBytes)) !=
      cudaSuccess)
    return e;
  // programmatic dependent launch: the CTAs take the SMs as those of the
  // kernel before leave, and wait for it (in the kernel) before reading
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t scfg = {};
  scfg.gridDim = dim3(num_sms());
  scfg.blockDim = dim3(kSThreads);
  scfg.dynamicSmemBytes = kSSmemBytes;
  scfg.stream = st;
  scfg.attrs = attr;
  scfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&scfg, k1, sp, tm_k, tm_v);
  count_launch();
  if (e != cudaSuccess) return e;

  constexpr int F = D * D + D;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.B * p.H, (F / 4 + kReduceThreads - 1) / kReduceThreads);
  // Lean blocks (32 registers, up to 16 an SM) for a grid of at most one block
  // per SM, which then waits beside the state CTAs, and for a grid that the
  // wide blocks (16 loads in flight, 116 registers) would run in more than one
  // wave; wide blocks when they fit one wave.  Measured at D = 128 on 32
  // ragged sequences (8448 blocks): 562.8 -> 540.1 us per forward with lean
  // blocks; with 288 and 576 blocks lean ones were 6.5-9.4 us slower.
  static const int wide_per_sm = [] {
    int n = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, tc_reduce_kernel<D, false>,
                                                      kReduceThreads, 0) != cudaSuccess) {
      (void)cudaGetLastError();
      n = 1;
    }
    return n;
  }();
  const long long nblk = (long long)cfg.gridDim.x * cfg.gridDim.y;
  const bool lean = nblk <= num_sms() || nblk > (long long)wide_per_sm * num_sms();
  if (lean) {  // the SMs keep the state kernel's shared-memory split for the lean blocks
    static std::once_flag carve;
    std::call_once(carve, [] {  // a hint: if it is refused, the launch goes on without it
      if (cudaFuncSetAttribute(tc_reduce_kernel<D, true>,
                               cudaFuncAttributePreferredSharedMemoryCarveout,
                               (int)cudaSharedmemCarveoutMaxShared) != cudaSuccess)
        (void)cudaGetLastError();
    });
  }
  cfg.blockDim = dim3(kReduceThreads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = st;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, lean ? tc_reduce_kernel<D, true> : tc_reduce_kernel<D, false>,
                         (const float *)sp.records, p.seq_lens, state, gate_stats, p.B, p.H,
                         p.N, num_sms());
  count_launch();
  return e;
}

template <int D>
cudaError_t run_readout(const Problem &p, const void *q, const void *og, const float *conv_w,
                        const float *norm_w, const float *state, void *o, cudaStream_t st,
                        bool after_state, bool f32_out) {
  using C = ReadoutCfg<D>;
  CUtensorMap tm_og, tm_o, tm_q;
  cudaError_t e = make_bnhd_map(&tm_og, og, p.B, p.N, p.H, D, kRTok);
  if (e != cudaSuccess) return e;
  if ((e = make_bnhd_map(&tm_o, o, p.B, p.N, p.H, D, 32)) != cudaSuccess) return e;  // a quarter
  if ((e = make_bnhd_map(&tm_q, q, p.B, p.N, p.H, D, kRQRows)) != cudaSuccess)
    return e;
  ReadoutParams rp;
  rp.q = (const __nv_bfloat16 *)q;
  rp.conv_w = conv_w;
  rp.norm_w = norm_w;
  rp.state = state;
  rp.seq_lens = p.seq_lens;
  rp.o = (__nv_bfloat16 *)o;
  rp.o32 = (float *)o;
  rp.B = p.B;
  rp.H = p.H;
  rp.N = p.N;
  rp.eps = kRmsEps;
  rp.wait_late = after_state ? 1 : 0;
  rp.flags = p.flags;
  auto kern = f32_out ? tc_readout_kernel<D, false, true>
                      : (p.flags ? tc_readout_kernel<D, true, false> : tc_readout_kernel<D, false, false>);
  if ((e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmem)) !=
      cudaSuccess)
    return e;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.gridDim = dim3(num_sms());
  cfg.blockDim = dim3(kRThreads);
  cfg.dynamicSmemBytes = C::kSmem;
  cfg.stream = st;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, kern, rp, tm_og, tm_o, tm_q);
  count_launch();
  return e;
}

}  // namespace

bool tc_supports(const Problem &p) {
  if (p.dtype != GBLA_BF16) return false;
  if (p.D != 64 && p.D != 128) return false;
  if (p.B > kMaxBatch) return false;
  // sequences of at most 2^23 tokens (the combination's scale factors of one
  // sequence fit in shared memory)
  if (p.N > (1 << 23)) return false;
  // stage indices are ints: B * HG * ceil(N / 64) stages at most
  if ((long long)p.B * ((p.H + kGroupCh / p.D - 1) / (kGroupCh / p.D)) *
          (((long long)p.N + kSTok - 1) / kSTok) > (1ll << 30))
    return false;
  if ((long long)p.B * p.H > 2147483647ll / 4) return false;
  if (p.H < kGroupCh / p.D) return false;  // the state tiles span a whole head group
  return device_info().sm103 && encode_fn() != nullptr;
}

size_t tc_workspace_bytes(const Problem &p) { return records_bytes(p) + 256; }

cudaError_t tc_state(const Problem &p, const void *k, const void *v, const void *gate,
                     const float *conv_w, void *ws, float *state, cudaStream_t st,
                     float2 *gate_stats) {
  switch (p.D) {
    case 64: return run_state<64>(p, k, v, gate, conv_w, ws, state, st, gate_stats);
    case 128: return run_state<128>(p, k, v, gate, conv_w, ws, state, st, gate_stats);
  }
  return cudaErrorInvalidValue;
}

cudaError_t tc_readout(const Problem &p, const void *q, const void *og, const float *conv_w,
                       const float *norm_w, const float *state, void *o, cudaStream_t st,
                       bool after_state, bool f32_out) {
  if (f32_out && p.flags) return cudaErrorInvalidValue;  // the debug output is the full core's
  switch (p.D) {
    case 64: return run_readout<64>(p, q, og, conv_w, norm_w, state, o, st, after_state, f32_out);
    case 128:
      return run_readout<128>(p, q, og, conv_w, norm_w, state, o, st, after_state, f32_out);
  }
  return cudaErrorInvalidValue;
}

unsigned tc_device_error(bool reset) {
  unsigned v = 0;
  if (cudaMemcpyFromSymbol(&v, g_tc_error, sizeof(v)) != cudaSuccess) return 0xFFFFFFFFu;
  if (reset) {
    const unsigned z = 0;
    if (cudaMemcpyToSymbol(g_tc_error, &z, sizeof(z)) != cudaSuccess) return 0xFFFFFFFFu;
  }
  return v;
}

}  // namespace gbla
