// Tensor-core (tcgen05 + TMEM + TMA) kernels of the GBLA core for bf16 inputs,
// D in {64, 128}.  Three kernels, launched back to back on one stream:
//
//  tc_state_kernel   (Sec. 2.1 item 1 and item 2, k/v side)
//      Persistent; one CTA per SM.  Each (batch, group of 128/D heads) sequence
//      is cut into chunks of S tokens and every CTA takes a contiguous range of
//      chunks, so work is balanced whatever the sequence lengths.  Per chunk:
//      a pre-pass over the gate logits gives the chunk maximum m and the
//      weights w_j = exp(a_j - m); eight producer warps then stream k and v
//      from HBM with 128-bit loads, run the causal Conv1D (sliding window in
//      registers, packed f32x2 FMAs), phi and the gate weight, and write
//      K^ (bf16) and V~ as a bf16 hi/lo pair into 128B-swizzled MN-major
//      tiles; one thread issues tcgen05.mma (M = N = 128, K = 16, fp32
//      accumulation in TMEM): D += K^T V~_hi + K^T V~_lo.  The diagonal
//      D x D blocks of the accumulator are the per-head partial states S_c;
//      z_c, m_c and l_c = sum w_j complete each partial record.
//  tc_reduce_kernel  fixed-order, max-rescaled combination of the partial
//      records into S = K^T V~ and z = K^T 1 with the softmax gate.
//  tc_readout_kernel (Sec. 2.1 item 2 readout and item 3)
//      Persistent; 128-token tiles of one (batch, head).  Four producer warps
//      compute phi(Conv1D(q)) into a K-major bf16 tile; one thread issues
//      tcgen05.mma against [S | z] (bf16 hi + lo, N = D + 16), giving
//      phi(q~)^T S and phi(q~)^T z per token in TMEM; four epilogue warps
//      (one token row per thread) divide, apply RMSNorm, the norm weight and
//      SiLU(out_gate) (out_gate tile brought in by TMA) and write o in place
//      of the out_gate tile, which TMA stores back.
//
// Why V~ is split into hi + lo: V~ = Conv1D(v) is not representable in bf16,
// and its rounding error does not average out, because O is a heavily
// cancelling weighted mean of the v rows (|O| shrinks like 1/sqrt(L) while the
// rows stay O(1)); V~_hi + V~_lo carries 16 significant bits.  K^ only weights
// the mean, so bf16 is enough there, and z sums the same rounded K^ the MMA sees.
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
constexpr int kSWarps = 8;                      // producer warps
constexpr int kSThreads = (kSWarps + 1) * 32;   // + 1 MMA warp
constexpr int kSProd = kSWarps * 32;
constexpr int kSTok = 32;                       // tokens per pipeline stage
constexpr int kSStages = 4;
constexpr int kSSub = 16;                       // sub-streams (half-warps)
constexpr int kSTokPerSub = kSTok / kSSub;      // 2
constexpr int kChunkMax = 2048;                 // longest chunk (tokens)
constexpr int kMaxChunksPerSeq = 4096;
constexpr int kSBlock = kSTok * 128;            // 64-channel MN block: 32 rows x 128 B
constexpr int kSOp = 2 * kSBlock;               // one 128-channel operand
constexpr int kSStageBytes = 3 * kSOp;          // A, B_hi, B_lo
constexpr uint32_t kSTmemCols = 128;
constexpr int kSPrefetch = 12;                  // L2 prefetch distance (tokens)

constexpr int kMaxBatch = 2048;

// Shared-memory map of the state kernel (offsets from a 1024-aligned base).
constexpr int kSOffStages = 0;
constexpr int kSOffGate = kSStages * kSStageBytes;               // float [2][kChunkMax]
constexpr int kSOffZred = kSOffGate + 2 * kChunkMax * 4;         // float [kSSub][128]
constexpr int kSOffRed = kSOffZred + kSSub * kGroupCh * 4;       // float [96]
constexpr int kSOffPre = kSOffRed + 96 * 4;                      // int [kMaxBatch + 1]
constexpr int kSOffBar = kSOffPre + ((kMaxBatch + 1) * 4 + 15) / 16 * 16;
constexpr int kSBarCount = 2 * kSStages + 2;                      // full, empty, done, final
constexpr int kSOffMisc = kSOffBar + kSBarCount * 8;              // tmem addr, abort flag
constexpr int kSSmemBytes = kSOffMisc + 16 + 1024;                // + alignment slack

// ------------------------------------------------------------------ readout
constexpr int kRTok = 128;                      // tokens per tile (MMA M)
constexpr int kRThreads = 10 * 32;              // 4 producer, 4 epilogue, MMA, TMA warps
constexpr int kRAStages = 2;
constexpr int kRAccBufs = 2;

template <int D>
struct ReadoutCfg {
  static constexpr int NR = D + 16;                       // MMA N: D columns of S, z, zeros
  static constexpr int KB = D / 64;                       // 64-element K blocks
  static constexpr int kABytes = kRTok * D * 2;           // one A tile
  static constexpr int kBBytes = NR * D * 2;              // one of B_hi / B_lo
  static constexpr int kOgStages = D == 128 ? 2 : 3;
  static constexpr int kOgBytes = kRTok * D * 2;
  static constexpr int kOffA = 0;
  static constexpr int kOffBhi = kOffA + kRAStages * kABytes;
  static constexpr int kOffBlo = kOffBhi + kBBytes;
  static constexpr int kOffOg = kOffBlo + kBBytes;
  static constexpr int kOffPre = kOffOg + kOgStages * kOgBytes;  // int [kMaxBatch + 1]
  static constexpr int kOffBar = kOffPre + ((kMaxBatch + 1) * 4 + 15) / 16 * 16;
  // a_full[2], a_empty[2], og_full[S], og_empty[S], acc_full[2], acc_empty[2],
  // b_full, b_free, final
  static constexpr int kBars = 2 * kRAStages + 2 * kOgStages + 2 * kRAccBufs + 3;
  static constexpr int kOffMisc = kOffBar + kBars * 8;
  static constexpr int kSmem = kOffMisc + 16 + 1024;
  static constexpr uint32_t kAccStride = NR <= 128 ? 128 : 256;  // column offset of buffer 1
  static constexpr uint32_t kTmemCols = kAccStride + NR <= 256 ? 256 : 512;
  static constexpr uint32_t kIdesc = idesc_bf16_f32(kRTok, NR, 0, 0);
  static_assert(kSmem <= 227 * 1024, "readout shared memory");
};

__device__ __forceinline__ void report_error(unsigned code, volatile int *abort_flag) {
  atomicOr(&g_tc_error, code);
  *abort_flag = 1;
}

__device__ __forceinline__ int clamp_len(const int32_t *seq_lens, int b, int N) {
  if (seq_lens == nullptr) return N;
  int L = seq_lens[b];
  return L < 0 ? 0 : (L > N ? N : L);
}

// Exclusive prefix over b of count(b) into pre[0..B], computed by the `nthr`
// threads with tid < nthr (a multiple of 32, at most 256).  Ends with a named
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

// phi(x) = elu(x) + 1 = exp(min(x, 0)) + max(x, 0)
__device__ __forceinline__ float phi_fast(float x) {
  return __expf(fminf(x, 0.f)) + fmaxf(x, 0.f);
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

// Causal Conv1D of two channels: taps 0..2 on x[t-3..t-1], tap 3 on x[t].
__device__ __forceinline__ float2 conv2(const float (&w)[4][8], const float (&xm)[3][8],
                                        const float (&x)[8], int i) {
  float2 a = __fmul2_rn(make_float2(w[0][i], w[0][i + 1]), make_float2(xm[0][i], xm[0][i + 1]));
  a = __ffma2_rn(make_float2(w[1][i], w[1][i + 1]), make_float2(xm[1][i], xm[1][i + 1]), a);
  a = __ffma2_rn(make_float2(w[2][i], w[2][i + 1]), make_float2(xm[2][i], xm[2][i + 1]), a);
  a = __ffma2_rn(make_float2(w[3][i], w[3][i + 1]), make_float2(x[i], x[i + 1]), a);
  return a;
}

__device__ __forceinline__ void slide(float (&xm)[3][8], const float (&x)[8]) {
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    xm[0][i] = xm[1][i];
    xm[1][i] = xm[2][i];
    xm[2][i] = x[i];
  }
}

// ===================================================================== state
struct StateParams {
  const __nv_bfloat16 *k, *v, *gate;
  const float *conv_w;
  const int32_t *seq_lens;
  float *records;        // [chunks][G][D*D + D + 4]: S, z, m, l, 2 pad
  int32_t *chunk_pre;    // [B + 1] chunk prefix (written by CTA 0)
  int B, H, N, S, HG;
};

template <int D>
__global__ void __launch_bounds__(kSThreads, 1) tc_state_kernel(const StateParams p) {
  constexpr int G = kGroupCh / D;
  constexpr int REC = D * D + D + 4;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  float *gw = (float *)(smem + kSOffGate);           // [G][kChunkMax]
  float *zred = (float *)(smem + kSOffZred);         // [kSSub][128]
  float *red = (float *)(smem + kSOffRed);           // [0,32) max, [32,64) sum, 64+ m, 68+ l
  int *pre = (int *)(smem + kSOffPre);
  uint64_t *bars = (uint64_t *)(smem + kSOffBar);
  uint64_t *full = bars, *empty = bars + kSStages, *done = bars + 2 * kSStages,
           *fin = bars + 2 * kSStages + 1;
  uint32_t *tmem_slot = (uint32_t *)(smem + kSOffMisc);
  volatile int *abort_flag = (volatile int *)(smem + kSOffMisc + 4);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int B = p.B, H = p.H, N = p.N, S = p.S, HG = p.HG;

  if (tid == 0) {
    *abort_flag = 0;
    for (int i = 0; i < kSBarCount; ++i) mbar_init(&bars[i], i < kSStages ? kSWarps : 1);
    fence_mbar_init();
  }
  // Chunk prefix over the batch (producer threads), shared by all roles.
  if (warp < kSWarps) {
    prefix_counts(pre, B, tid, kSProd, 1, (int *)red, [&](int b) {
      const int L = clamp_len(p.seq_lens, b, N);
      return HG * ((L + S - 1) / S);
    });
  }
  __syncthreads();
  const int K = pre[B];
  if (blockIdx.x == 0)
    for (int i = tid; i <= B; i += kSThreads) p.chunk_pre[i] = pre[i];
  const long long c0 = (long long)K * blockIdx.x / gridDim.x;
  const long long c1 = (long long)K * (blockIdx.x + 1) / gridDim.x;
  grid_dep_launch();
  if (c0 >= c1) return;  // no chunks for this CTA

  if (warp == kSWarps) tmem_alloc(tmem_slot, kSTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp < kSWarps) {
    // ------------------------------------------------------------ producers
    const int half = lane >> 4, c = lane & 15;       // c: 8-channel chunk of the group
    const int sub = warp * 2 + half;                 // sub-stream 0..15
    const int hh = (8 * c) / D, d0 = 8 * c - D * hh; // head within group, first channel
    const int blk = c >> 3, cc = c & 7;              // MN block, 16-byte chunk in block
    uint32_t gs = 0;                                 // stage counter across chunks
    int nchunk = 0;
    for (long long kk = c0; kk < c1; ++kk, ++nchunk) {
      const int k = (int)kk;
      const int b = find_batch(pre, B, k);
      const int L = clamp_len(p.seq_lens, b, N);
      const int nck = (L + S - 1) / S;
      const int r = k - pre[b];
      const int hg = r / nck, j = r % nck;
      const int t0 = j * S, t1 = min(t0 + S, L), n = t1 - t0;
      const int hbase = hg * G;

      // Gate pre-pass: chunk maximum and weights per head (thread's head = tid % G).
      {
        const int myh = tid % G;
        const int hglob = hbase + myh;
        float m = -INFINITY;
        for (int idx = tid; idx < n * G; idx += kSProd) {
          const int tt = idx / G;
          float a = -INFINITY;
          if (hglob < H) a = __bfloat162float(p.gate[((size_t)b * N + t0 + tt) * H + hglob]);
          gw[myh * kChunkMax + tt] = a;
          m = fmaxf(m, a);
        }
#pragma unroll
        for (int o = 16; o >= G; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
        if (lane < G) red[warp * 4 + lane] = m;
        named_barrier(1, kSProd);
        float M = red[myh];
        for (int w = 1; w < kSWarps; ++w) M = fmaxf(M, red[w * 4 + myh]);
        float l = 0.f;
        for (int idx = tid; idx < n * G; idx += kSProd) {
          const int tt = idx / G;
          const float a = gw[myh * kChunkMax + tt];
          const float w = (hglob < H) ? __expf(a - M) : 0.f;
          gw[myh * kChunkMax + tt] = w;
          l += w;
        }
#pragma unroll
        for (int o = 16; o >= G; o >>= 1) l += __shfl_xor_sync(0xffffffffu, l, o);
        if (lane < G) red[32 + warp * 4 + lane] = l;
        named_barrier(1, kSProd);
        if (tid < G) {  // m and l of this chunk, per head, for the records
          float lt = 0.f;
          for (int w = 0; w < kSWarps; ++w) lt += red[32 + w * 4 + tid];
          red[64 + tid] = M;
          red[68 + tid] = lt;
        }
      }

      // This thread's channels: group channels [8c, 8c+8) of k and v.
      const int h = hbase + hh;
      const bool hv = h < H;
      const size_t rs = (size_t)H * D;  // token stride
      const __nv_bfloat16 *kp = p.k + ((size_t)b * N * H + (hv ? h : 0)) * D + d0;
      const __nv_bfloat16 *vp = p.v + ((size_t)b * N * H + (hv ? h : 0)) * D + d0;
      float wk[4][8], wv[4][8];
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          wk[q][i] = hv ? p.conv_w[((size_t)(1 * H + h) * D + d0 + i) * 4 + q] : 0.f;
          wv[q][i] = hv ? p.conv_w[((size_t)(2 * H + h) * D + d0 + i) * 4 + q] : 0.f;
        }
      const int s0 = t0 + (int)((long long)n * sub / kSSub);
      const int s1 = t0 + (int)((long long)n * (sub + 1) / kSSub);
      float km[3][8], vm[3][8];  // sliding windows x[t-3], x[t-2], x[t-1]
#pragma unroll
      for (int q = 0; q < 3; ++q) {
        const int t = s0 - 3 + q;
        uint4 rk = make_uint4(0, 0, 0, 0), rv = rk;
        if (hv && t >= 0 && s0 < s1) {
          rk = ldg_nc_v4(kp + (size_t)t * rs);
          rv = ldg_nc_v4(vp + (size_t)t * rs);
        }
        float xk[8], xv[8];
        unpack8(rk, xk);
        unpack8(rv, xv);
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          km[q][i] = xk[i];
          vm[q][i] = xv[i];
        }
      }
      float zacc[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) zacc[i] = 0.f;
      const float *gwh = gw + hh * kChunkMax;
      const int nst = ((n + kSSub - 1) / kSSub + kSTokPerSub - 1) / kSTokPerSub;
      const uint32_t grow_bytes = (uint32_t)(min(G, H - hbase) * D * 2);
      const __nv_bfloat16 *kgrp = p.k + ((size_t)b * N * H + hbase) * D;
      const __nv_bfloat16 *vgrp = p.v + ((size_t)b * N * H + hbase) * D;
      if (c == 0)  // warm L2 with the first tokens of this sub-stream
        for (int t = s0; t < min(s1, s0 + kSPrefetch); ++t) {
          prefetch_l2(kgrp + (size_t)t * rs, grow_bytes);
          prefetch_l2(vgrp + (size_t)t * rs, grow_bytes);
        }

      for (int it = 0; it < nst; ++it, ++gs) {
        const int s = gs % kSStages;
        if (!mbar_wait(&empty[s], ((gs / kSStages) & 1) ^ 1, abort_flag) && !*abort_flag)
          report_error(1, abort_flag);
        const uint32_t stage = smem_u32(smem + kSOffStages + s * kSStageBytes);
        uint4 rk[kSTokPerSub], rv[kSTokPerSub];
#pragma unroll
        for (int u = 0; u < kSTokPerSub; ++u) {
          const int t = s0 + it * kSTokPerSub + u;
          rk[u] = make_uint4(0, 0, 0, 0);
          rv[u] = rk[u];
          if (hv && t < s1) {
            rk[u] = ldg_nc_v4(kp + (size_t)t * rs);
            rv[u] = ldg_nc_v4(vp + (size_t)t * rs);
          }
          const int tp = t + kSPrefetch;
          if (c == 0 && tp < s1) {
            prefetch_l2(kgrp + (size_t)tp * rs, grow_bytes);
            prefetch_l2(vgrp + (size_t)tp * rs, grow_bytes);
          }
        }
#pragma unroll
        for (int u = 0; u < kSTokPerSub; ++u) {
          const int t = s0 + it * kSTokPerSub + u;
          const bool valid = hv && t < s1;
          float xk[8], xv[8];
          unpack8(rk[u], xk);
          unpack8(rv[u], xv);
          const float wgt = valid ? gwh[t - t0] : 0.f;
          uint32_t pk[4], ph[4], pl[4];
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const float2 ck = conv2(wk, km, xk, 2 * i);
            const float2 cv = conv2(wv, vm, xv, 2 * i);
            // K^ = w * phi(k~); rows past the sub-stream end are zero
            const float k0 = valid ? wgt * phi_fast(ck.x) : 0.f;
            const float k1 = valid ? wgt * phi_fast(ck.y) : 0.f;
            pk[i] = f2_to_bf2(k0, k1);
            const float2 kr = bf2_to_f2(pk[i]);  // z sums exactly what the MMA sees
            zacc[2 * i] += kr.x;
            zacc[2 * i + 1] += kr.y;
            const float v0 = valid ? cv.x : 0.f, v1 = valid ? cv.y : 0.f;
            ph[i] = f2_to_bf2(v0, v1);
            const float2 vr = bf2_to_f2(ph[i]);
            pl[i] = f2_to_bf2(v0 - vr.x, v1 - vr.y);
          }
          slide(km, xk);
          slide(vm, xv);
          // row of this token in the stage; MN-major, 128-byte swizzle
          const int row = sub * kSTokPerSub + u;
          const uint32_t sa = stage + blk * kSBlock + (row >> 3) * 1024 + (row & 7) * 128 +
                              ((cc ^ (row & 7)) << 4);
          sts_v4(sa, make_uint4(pk[0], pk[1], pk[2], pk[3]));
          sts_v4(sa + kSOp, make_uint4(ph[0], ph[1], ph[2], ph[3]));
          sts_v4(sa + 2 * kSOp, make_uint4(pl[0], pl[1], pl[2], pl[3]));
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(&full[s]);
      }

      // z of this chunk: the 16 sub-streams summed in a fixed order.
#pragma unroll
      for (int i = 0; i < 8; ++i) zred[sub * kGroupCh + 8 * c + i] = zacc[i];
      named_barrier(1, kSProd);
      float zsum = 0.f;
      if (tid < kGroupCh)
        for (int q = 0; q < kSSub; ++q) zsum += zred[q * kGroupCh + tid];

      // Wait for this chunk's accumulator, then write the partial records.
      if (!mbar_wait(done, nchunk & 1, abort_flag) && !*abort_flag) report_error(2, abort_flag);
      tc_fence_after();
      {
        const int q4 = warp & 3, colhalf = warp >> 2;
        const int ch = 32 * q4 + lane;               // TMEM lane = group channel (row of S)
        const int hh2 = ch / D, d = ch - D * hh2;
        const int col0 = D * hh2 + colhalf * (D / 2);
        const bool ok2 = hbase + hh2 < H;
        float *srow = p.records + ((size_t)k * G + hh2) * REC + (size_t)d * D + colhalf * (D / 2);
#pragma unroll
        for (int cb = 0; cb < D / 2; cb += 16) {
          float vals[16];
          tmem_ld16(tmem + ((uint32_t)(32 * q4) << 16) + (uint32_t)(col0 + cb), vals);
          tmem_ld_wait();
          if (ok2) {
            float4 *dst = (float4 *)(srow + cb);
#pragma unroll
            for (int i = 0; i < 4; ++i)
              dst[i] = make_float4(vals[4 * i], vals[4 * i + 1], vals[4 * i + 2], vals[4 * i + 3]);
          }
        }
        if (tid < kGroupCh) {
          const int hz = tid / D, dz = tid - D * hz;
          if (hbase + hz < H) {
            float *rz = p.records + ((size_t)k * G + hz) * REC;
            rz[D * D + dz] = zsum;
            if (dz == 0) {
              rz[D * D + D] = red[64 + hz];
              rz[D * D + D + 1] = red[68 + hz];
            }
          }
        }
      }
      tc_fence_before();
      named_barrier(1, kSProd);  // accumulator drained before the next chunk's MMAs
    }
  } else if (lane == 0) {
    // ------------------------------------------------------------ MMA issuer
    constexpr uint32_t idesc = idesc_bf16_f32(128, 128, 1, 1);
    uint32_t gs = 0;
    bool ok = true;
    for (long long kk = c0; kk < c1 && ok; ++kk) {
      const int k = (int)kk;
      const int b = find_batch(pre, B, k);
      const int L = clamp_len(p.seq_lens, b, N);
      const int nck = (L + S - 1) / S;
      const int j = (k - pre[b]) % nck;
      const int n = min(S, L - j * S);
      const int nst = ((n + kSSub - 1) / kSSub + kSTokPerSub - 1) / kSTokPerSub;
      for (int it = 0; it < nst; ++it, ++gs) {
        const int s = gs % kSStages;
        if (!mbar_wait(&full[s], (gs / kSStages) & 1, abort_flag)) {
          if (!*abort_flag) report_error(4, abort_flag);
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t base = smem_u32(smem + kSOffStages + s * kSStageBytes);
#pragma unroll
        for (int k16 = 0; k16 < kSTok / 16; ++k16) {
          const uint32_t o = k16 * 2048;
          const uint64_t ad = sw128_desc(base + o, kSBlock, 1024);
          const uint64_t bh = sw128_desc(base + kSOp + o, kSBlock, 1024);
          const uint64_t bl = sw128_desc(base + 2 * kSOp + o, kSBlock, 1024);
          mma_bf16(tmem, ad, bh, idesc, (it | k16) != 0);
          mma_bf16(tmem, ad, bl, idesc, 1);
        }
        mma_commit(&empty[s]);
      }
      if (ok) mma_commit(done);
    }
    mma_commit(fin);  // every MMA issued above has completed once this arrives
    if (!mbar_wait(fin, 0, nullptr)) report_error(8, abort_flag);
  }
  __syncthreads();
  if (warp == kSWarps) {
    tc_fence_after();
    tmem_dealloc(tmem, kSTmemCols);
  }
}

// Fixed-order combination of the chunk records of one (b, h).
template <int D>
__global__ void __launch_bounds__(256) tc_reduce_kernel(const float *__restrict__ records,
                                                         const int32_t *__restrict__ chunk_pre,
                                                         const int32_t *__restrict__ seq_lens,
                                                         float *__restrict__ state, int B, int H,
                                                         int N, int S) {
  constexpr int G = kGroupCh / D;
  constexpr int REC = D * D + D + 4;
  constexpr int F = D * D + D;
  __shared__ float s_scale[kMaxChunksPerSeq];
  __shared__ float s_l;
  grid_dep_wait();
  grid_dep_launch();
  const int bh = blockIdx.x;
  const int b = bh / H, h = bh % H;
  const int hg = h / G, hh = h % G;
  const int L = clamp_len(seq_lens, b, N);
  const int nck = (L + S - 1) / S;
  const int k0 = chunk_pre[b] + hg * nck;
  const float *rec0 = records + ((size_t)k0 * G + hh) * REC;
  const size_t rstride = (size_t)G * REC;
  if (threadIdx.x < 32) {
    float M = -INFINITY;
    for (int j = threadIdx.x; j < nck; j += 32) M = fmaxf(M, rec0[j * rstride + F]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
    for (int j = threadIdx.x; j < nck; j += 32) s_scale[j] = __expf(rec0[j * rstride + F] - M);
    __syncwarp();
    if (threadIdx.x == 0) {
      float l = 0.f;
      for (int j = 0; j < nck; ++j) l = fmaf(s_scale[j], rec0[j * rstride + F + 1], l);
      s_l = l;
    }
  }
  __syncthreads();
  const int e = blockIdx.y * 256 + threadIdx.x;
  if (e >= F) return;
  float acc = 0.f;
  for (int j = 0; j < nck; ++j) acc = fmaf(s_scale[j], rec0[j * rstride + e], acc);
  state[(size_t)bh * F + e] = s_l > 0.f ? acc / s_l : 0.f;
}

// ===================================================================== readout
struct ReadoutParams {
  const __nv_bfloat16 *q;
  const float *conv_w, *norm_w, *state;
  const int32_t *seq_lens;
  __nv_bfloat16 *o;
  int B, H, N;
  float eps;
};

template <int D>
__global__ void __launch_bounds__(kRThreads, 1)
    tc_readout_kernel(const ReadoutParams p, const __grid_constant__ CUtensorMap tm_og,
                      const __grid_constant__ CUtensorMap tm_o) {
  using C = ReadoutCfg<D>;
  constexpr int NR = C::NR;
  constexpr int OGS = C::kOgStages;
  constexpr int F = D * D + D;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  int *pre = (int *)(smem + C::kOffPre);
  uint64_t *bars = (uint64_t *)(smem + C::kOffBar);
  uint64_t *a_full = bars, *a_empty = bars + 2, *og_full = bars + 4, *og_empty = og_full + OGS,
           *acc_full = og_empty + OGS, *acc_empty = acc_full + 2, *b_full = acc_empty + 2,
           *b_free = b_full + 1, *fin = b_free + 1;
  uint32_t *tmem_slot = (uint32_t *)(smem + C::kOffMisc);
  volatile int *abort_flag = (volatile int *)(smem + C::kOffMisc + 4);
  __shared__ int s_tot[8];

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int B = p.B, H = p.H, N = p.N;

  if (tid == 0) {
    *abort_flag = 0;
    mbar_init(&a_full[0], 4);
    mbar_init(&a_full[1], 4);
    mbar_init(&a_empty[0], 1);
    mbar_init(&a_empty[1], 1);
    for (int i = 0; i < OGS; ++i) {
      mbar_init(&og_full[i], 1);
      mbar_init(&og_empty[i], 1);
    }
    mbar_init(&acc_full[0], 1);
    mbar_init(&acc_full[1], 1);
    mbar_init(&acc_empty[0], 4);
    mbar_init(&acc_empty[1], 4);
    mbar_init(b_full, 4);
    mbar_init(b_free, 1);
    mbar_init(fin, 1);
    fence_mbar_init();
  }
  if (warp == 9 && lane == 0) {
    tma_prefetch_desc(&tm_og);
    tma_prefetch_desc(&tm_o);
  }
  // Everything below may read what earlier work on the stream wrote.
  grid_dep_wait();
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
  if (warp == 8) tmem_alloc(tmem_slot, C::kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  // Tile -> (b, h, first token, valid rows)
  auto tile_of = [&](long long ii, int &b, int &h, int &r0, int &nrow) {
    const int i = (int)ii;
    b = find_batch(pre, B, i);
    const int L = clamp_len(p.seq_lens, b, N);
    const int nt = (L + kRTok - 1) / kRTok;
    const int r = i - pre[b];
    h = r / nt;
    r0 = (r % nt) * kRTok;
    nrow = min(kRTok, L - r0);
  };

  if (warp < 4) {
    // ------------------------------------------------------------ producers: phi(conv(q))
    constexpr int TPR = D / 8;            // threads per token row
    constexpr int STREAMS = 128 / TPR;    // sub-streams per tile
    constexpr int TPS = kRTok / STREAMS;  // tokens per sub-stream
    const int c = tid % TPR, stream = tid / TPR;
    const int kb = c >> 3, cc = c & 7;
    int cur_b = -1, cur_h = -1, nbh = 0;
    float wq[4][8];
    for (long long ii = i0; ii < i1; ++ii) {
      int b, h, r0, nrow;
      tile_of(ii, b, h, r0, nrow);
      const int li = (int)(ii - i0);
      if (b != cur_b || h != cur_h) {
        // New (b, h): rebuild B = [S | z | 0] as bf16 hi/lo, K-major, 128B swizzle,
        // once the MMAs that read the previous one have completed.
        if (nbh > 0 && !mbar_wait(b_free, (nbh - 1) & 1, abort_flag) && !*abort_flag)
          report_error(16, abort_flag);
        const float *st = p.state + ((size_t)b * H + h) * F;
        for (int item = tid; item < NR * (D / 8); item += 128) {
          const int e = item % NR, ck = item / NR;  // row e of B, 8-element K chunk ck
          float vals[8];
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const int d = 8 * ck + i;
            vals[i] = e < D ? st[(size_t)d * D + e] : (e == D ? st[D * D + d] : 0.f);
          }
          uint32_t hi[4], lo[4];
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            hi[i] = f2_to_bf2(vals[2 * i], vals[2 * i + 1]);
            const float2 hr = bf2_to_f2(hi[i]);
            lo[i] = f2_to_bf2(vals[2 * i] - hr.x, vals[2 * i + 1] - hr.y);
          }
          const int kbk = ck >> 3, ckk = ck & 7;
          const uint32_t off = kbk * (NR * 128) + (e >> 3) * 1024 + (e & 7) * 128 +
                               ((ckk ^ (e & 7)) << 4);
          sts_v4(smem_u32(smem + C::kOffBhi) + off, make_uint4(hi[0], hi[1], hi[2], hi[3]));
          sts_v4(smem_u32(smem + C::kOffBlo) + off, make_uint4(lo[0], lo[1], lo[2], lo[3]));
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(b_full);
#pragma unroll
        for (int i = 0; i < 8; ++i)
#pragma unroll
          for (int q = 0; q < 4; ++q)
            wq[q][i] = p.conv_w[((size_t)(0 * H + h) * D + 8 * c + i) * 4 + q];
        cur_b = b;
        cur_h = h;
        ++nbh;
      }
      const int sa = li & 1;
      if (!mbar_wait(&a_empty[sa], ((li >> 1) & 1) ^ 1, abort_flag) && !*abort_flag)
        report_error(32, abort_flag);
      const size_t rs = (size_t)H * D;
      const __nv_bfloat16 *qp = p.q + ((size_t)b * N * H + h) * D + 8 * c;
      const int ts = r0 + stream * TPS;  // first token of this sub-stream
      uint4 raw[TPS + 3];
#pragma unroll
      for (int u = 0; u < TPS + 3; ++u) {
        const int t = ts - 3 + u;
        raw[u] = make_uint4(0, 0, 0, 0);
        if (t >= 0 && t < r0 + nrow) raw[u] = ldg_nc_v4(qp + (size_t)t * rs);
      }
      float xm[3][8];
#pragma unroll
      for (int u = 0; u < 3; ++u) {
        float x[8];
        unpack8(raw[u], x);
#pragma unroll
        for (int i = 0; i < 8; ++i) xm[u][i] = x[i];
      }
      const uint32_t abase = smem_u32(smem + C::kOffA + sa * C::kABytes);
#pragma unroll
      for (int u = 0; u < TPS; ++u) {
        const int row = stream * TPS + u;
        const bool valid = row < nrow;
        float x[8];
        unpack8(raw[u + 3], x);
        uint32_t pq[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const float2 a = conv2(wq, xm, x, 2 * i);
          pq[i] = valid ? f2_to_bf2(phi_fast(a.x), phi_fast(a.y)) : 0u;
        }
        slide(xm, x);
        const uint32_t off = kb * (kRTok * 128) + (row >> 3) * 1024 + (row & 7) * 128 +
                             ((cc ^ (row & 7)) << 4);
        sts_v4(abase + off, make_uint4(pq[0], pq[1], pq[2], pq[3]));
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&a_full[sa]);
    }
  } else if (warp < 8) {
    // ------------------------------------------------------------ epilogue
    const int q4 = warp & 3;
    const int row = 32 * q4 + lane;
    for (long long ii = i0; ii < i1; ++ii) {
      int b, h, r0, nrow;
      tile_of(ii, b, h, r0, nrow);
      const int li = (int)(ii - i0);
      const int ab = li & 1, so = li % OGS;
      if (!mbar_wait(&acc_full[ab], (li >> 1) & 1, abort_flag) && !*abort_flag)
        report_error(64, abort_flag);
      if (!mbar_wait(&og_full[so], (li / OGS) & 1, abort_flag) && !*abort_flag)
        report_error(64, abort_flag);
      tc_fence_after();
      const uint32_t tacc = tmem + ((uint32_t)(32 * q4) << 16) + ab * C::kAccStride;
      float den[16];
      tmem_ld16(tacc + D, den);
      tmem_ld_wait();
      const float inv = 1.f / den[0];
      float ss = 0.f;
#pragma unroll
      for (int cb = 0; cb < D; cb += 16) {
        float v[16];
        tmem_ld16(tacc + cb, v);
        tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const float O = v[i] * inv;
          ss = fmaf(O, O, ss);
        }
      }
      const float rr = rsqrtf(ss / (float)D + p.eps) * inv;  // y = acc * rr * w * silu(og)
      const float *nwh = p.norm_w + (size_t)h * D;
      uint8_t *ogt = smem + C::kOffOg + so * C::kOgBytes;
#pragma unroll
      for (int cb = 0; cb < D; cb += 16) {
        float v[16];
        tmem_ld16(tacc + cb, v);
        tmem_ld_wait();
#pragma unroll
        for (int half = 0; half < 2; ++half) {
          const int ch0 = cb + 8 * half;  // first channel of this 16-byte chunk
          const int kbo = ch0 >> 6, cco = (ch0 & 63) >> 3;
          const uint32_t sa = smem_u32(ogt) + kbo * (kRTok * 128) + (row >> 3) * 1024 +
                              (row & 7) * 128 + ((cco ^ (row & 7)) << 4);
          float g[8];
          unpack8(lds_v4(sa), g);
          const float4 w0 = __ldg((const float4 *)(nwh + ch0));
          const float4 w1 = __ldg((const float4 *)(nwh + ch0 + 4));
          const float wv8[8] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
          uint32_t outw[4];
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const float s0v = g[2 * i] / (1.f + __expf(-g[2 * i]));
            const float s1v = g[2 * i + 1] / (1.f + __expf(-g[2 * i + 1]));
            const float y0 = v[8 * half + 2 * i] * rr * wv8[2 * i] * s0v;
            const float y1 = v[8 * half + 2 * i + 1] * rr * wv8[2 * i + 1] * s1v;
            outw[i] = f2_to_bf2(y0, y1);
          }
          sts_v4(sa, make_uint4(outw[0], outw[1], outw[2], outw[3]));
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acc_empty[ab]);
      if (nrow == kRTok) {
        fence_proxy_async_smem();
        named_barrier(2, 128);
        if (warp == 4 && lane == 0) {
#pragma unroll
          for (int kbo = 0; kbo < C::KB; ++kbo)
            tma_store_4d(&tm_o, ogt + kbo * (kRTok * 128), kbo * 64, h, r0, b);
          tma_store_commit();
          tma_store_wait_read<0>();
          mbar_arrive(&og_empty[so]);
        }
      } else {
        // Ragged tail: rows past the sequence end must not be written.
        if (row < nrow) {
          __nv_bfloat16 *orow = p.o + (((size_t)b * N + r0 + row) * H + h) * D;
#pragma unroll
          for (int ch0 = 0; ch0 < D; ch0 += 8) {
            const int kbo = ch0 >> 6, cco = (ch0 & 63) >> 3;
            const uint32_t sa = smem_u32(ogt) + kbo * (kRTok * 128) + (row >> 3) * 1024 +
                                (row & 7) * 128 + ((cco ^ (row & 7)) << 4);
            *(uint4 *)(orow + ch0) = lds_v4(sa);
          }
        }
        named_barrier(2, 128);
        if (warp == 4 && lane == 0) mbar_arrive(&og_empty[so]);
      }
    }
    if (warp == 4 && lane == 0) tma_store_wait_all<0>();
  } else if (warp == 8) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      int cur_b = -1, cur_h = -1, nbh = 0;
      for (long long ii = i0; ii < i1; ++ii) {
        int b, h, r0, nrow;
        tile_of(ii, b, h, r0, nrow);
        const int li = (int)(ii - i0);
        bool ok = true;
        if (b != cur_b || h != cur_h) {
          ok = mbar_wait(b_full, nbh & 1, abort_flag);
          cur_b = b;
          cur_h = h;
          ++nbh;
        }
        const int sa = li & 1, ab = li & 1;
        ok = ok && mbar_wait(&a_full[sa], (li >> 1) & 1, abort_flag) &&
             mbar_wait(&acc_empty[ab], ((li >> 1) & 1) ^ 1, abort_flag);
        if (!ok) {
          if (!*abort_flag) report_error(128, abort_flag);
          break;
        }
        tc_fence_after();
        const uint32_t abase = smem_u32(smem + C::kOffA + sa * C::kABytes);
        const uint32_t bhi = smem_u32(smem + C::kOffBhi), blo = smem_u32(smem + C::kOffBlo);
        const uint32_t dacc = tmem + ab * C::kAccStride;
#pragma unroll
        for (int kbk = 0; kbk < C::KB; ++kbk)
#pragma unroll
          for (int k16 = 0; k16 < 4; ++k16) {
            const uint32_t ao = kbk * (kRTok * 128) + k16 * 32;
            const uint32_t bo = kbk * (NR * 128) + k16 * 32;
            const uint64_t ad = sw128_desc(abase + ao, 16, 1024);
            mma_bf16(dacc, ad, sw128_desc(bhi + bo, 16, 1024), C::kIdesc, (kbk | k16) != 0);
            mma_bf16(dacc, ad, sw128_desc(blo + bo, 16, 1024), C::kIdesc, 1);
          }
        mma_commit(&a_empty[sa]);
        mma_commit(&acc_full[ab]);
        // last tile of this (b, h) in this CTA: release B for the next rebuild
        bool last = ii + 1 >= i1;
        if (!last) {
          int b2, h2, r02, nrow2;
          tile_of(ii + 1, b2, h2, r02, nrow2);
          last = (b2 != b || h2 != h);
        }
        if (last) mma_commit(b_free);
      }
      mma_commit(fin);  // every MMA issued above has completed once this arrives
      if (!mbar_wait(fin, 0, nullptr)) report_error(256, abort_flag);
    }
  } else {
    // ------------------------------------------------------------ TMA loads of out_gate
    if (lane == 0) {
      for (long long ii = i0; ii < i1; ++ii) {
        int b, h, r0, nrow;
        tile_of(ii, b, h, r0, nrow);
        const int li = (int)(ii - i0);
        const int so = li % OGS;
        if (!mbar_wait(&og_empty[so], ((li / OGS) & 1) ^ 1, abort_flag)) {
          if (!*abort_flag) report_error(512, abort_flag);
          break;
        }
        uint8_t *dst = smem + C::kOffOg + so * C::kOgBytes;
        mbar_arrive_expect_tx(&og_full[so], C::kOgBytes);
#pragma unroll
        for (int kbo = 0; kbo < C::KB; ++kbo)
          tma_load_4d(dst + kbo * (kRTok * 128), &tm_og, &og_full[so], kbo * 64, h, r0, b);
      }
    }
  }
  __syncthreads();
  if (warp == 8) {
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

// 4-D map over a [B, N, H, D] bf16 tensor; box = 64 channels x 1 head x 128 tokens,
// 128-byte swizzle (the layout the readout's thread-per-row epilogue reads).
cudaError_t make_bnhd_map(CUtensorMap *m, const void *base, int B, int N, int H, int D) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return cudaErrorNotSupported;
  const cuuint64_t dims[4] = {(cuuint64_t)D, (cuuint64_t)H, (cuuint64_t)N, (cuuint64_t)B};
  const cuuint64_t strides[3] = {(cuuint64_t)D * 2, (cuuint64_t)H * D * 2,
                                 (cuuint64_t)N * H * D * 2};
  const cuuint32_t box[4] = {64, 1, kRTok, 1};
  const cuuint32_t estr[4] = {1, 1, 1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(base), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

int num_sms() {
  int dev = 0, n = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
  return n > 0 ? n : 1;
}

// Chunk length: about one chunk per SM over the padded problem, 32-aligned,
// within [256, kChunkMax], and at most kMaxChunksPerSeq chunks per sequence.
int chunk_len(const Problem &p) {
  const int G = kGroupCh / p.D;
  const int HG = (p.H + G - 1) / G;
  const long long work = (long long)p.B * HG * p.N;
  const int sms = num_sms();
  long long S = (work + sms - 1) / sms;
  S = (S + 31) / 32 * 32;
  S = S < 256 ? 256 : (S > kChunkMax ? kChunkMax : S);
  const long long Smin = ((long long)p.N + kMaxChunksPerSeq - 1) / kMaxChunksPerSeq;
  if (S < Smin) S = (Smin + 31) / 32 * 32;
  return (int)S;
}

size_t records_bytes(const Problem &p, int S) {
  const int G = kGroupCh / p.D;
  const int HG = (p.H + G - 1) / G;
  const size_t chunks = (size_t)p.B * HG * ((p.N + S - 1) / S);
  return chunks * G * ((size_t)p.D * p.D + p.D + 4) * sizeof(float);
}

template <int D>
cudaError_t run_state(const Problem &p, const void *k, const void *v, const void *gate,
                      const float *conv_w, void *ws, float *state, cudaStream_t st) {
  constexpr int G = kGroupCh / D;
  const int S = chunk_len(p);
  const size_t rb = records_bytes(p, S);
  StateParams sp;
  sp.k = (const __nv_bfloat16 *)k;
  sp.v = (const __nv_bfloat16 *)v;
  sp.gate = (const __nv_bfloat16 *)gate;
  sp.conv_w = conv_w;
  sp.seq_lens = p.seq_lens;
  sp.records = (float *)ws;
  sp.chunk_pre = (int32_t *)((char *)ws + rb);
  sp.B = p.B;
  sp.H = p.H;
  sp.N = p.N;
  sp.S = S;
  sp.HG = (p.H + G - 1) / G;
  auto k1 = tc_state_kernel<D>;
  cudaError_t e =
      cudaFuncSetAttribute(k1, cudaFuncAttributeMaxDynamicSharedMemorySize, kSSmemBytes);
  if (e != cudaSuccess) return e;
  k1<<<num_sms(), kSThreads, kSSmemBytes, st>>>(sp);
  count_launch();
  if ((e = cudaGetLastError()) != cudaSuccess) return e;

  constexpr int F = D * D + D;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.gridDim = dim3(p.B * p.H, (F + 255) / 256);
  cfg.blockDim = dim3(256);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = st;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, tc_reduce_kernel<D>, (const float *)sp.records,
                         (const int32_t *)sp.chunk_pre, p.seq_lens, state, p.B, p.H, p.N, S);
  count_launch();
  return e;
}

template <int D>
cudaError_t run_readout(const Problem &p, const void *q, const void *og, const float *conv_w,
                        const float *norm_w, const float *state, void *o, cudaStream_t st) {
  using C = ReadoutCfg<D>;
  CUtensorMap tm_og, tm_o;
  cudaError_t e = make_bnhd_map(&tm_og, og, p.B, p.N, p.H, D);
  if (e != cudaSuccess) return e;
  if ((e = make_bnhd_map(&tm_o, o, p.B, p.N, p.H, D)) != cudaSuccess) return e;
  ReadoutParams rp;
  rp.q = (const __nv_bfloat16 *)q;
  rp.conv_w = conv_w;
  rp.norm_w = norm_w;
  rp.state = state;
  rp.seq_lens = p.seq_lens;
  rp.o = (__nv_bfloat16 *)o;
  rp.B = p.B;
  rp.H = p.H;
  rp.N = p.N;
  rp.eps = kRmsEps;
  auto kern = tc_readout_kernel<D>;
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
  e = cudaLaunchKernelEx(&cfg, kern, rp, tm_og, tm_o);
  count_launch();
  return e;
}

}  // namespace

bool tc_supports(const Problem &p) {
  if (p.dtype != GBLA_BF16) return false;
  if (p.D != 64 && p.D != 128) return false;
  if (p.B > kMaxBatch) return false;
  if ((long long)p.N > (long long)kChunkMax * kMaxChunksPerSeq) return false;
  if ((long long)p.B * p.H > 2147483647ll / 4) return false;
  int dev = 0, major = 0, minor = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
  return major == 10 && minor == 3 && encode_fn() != nullptr;
}

size_t tc_workspace_bytes(const Problem &p) {
  return records_bytes(p, chunk_len(p)) + sizeof(int32_t) * (p.B + 1) + 256;
}

cudaError_t tc_state(const Problem &p, const void *k, const void *v, const void *gate,
                     const float *conv_w, void *ws, float *state, cudaStream_t st) {
  switch (p.D) {
    case 64: return run_state<64>(p, k, v, gate, conv_w, ws, state, st);
    case 128: return run_state<128>(p, k, v, gate, conv_w, ws, state, st);
  }
  return cudaErrorInvalidValue;
}

cudaError_t tc_readout(const Problem &p, const void *q, const void *og, const float *conv_w,
                       const float *norm_w, const float *state, void *o, cudaStream_t st) {
  switch (p.D) {
    case 64: return run_readout<64>(p, q, og, conv_w, norm_w, state, o, st);
    case 128: return run_readout<128>(p, q, og, conv_w, norm_w, state, o, st);
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
