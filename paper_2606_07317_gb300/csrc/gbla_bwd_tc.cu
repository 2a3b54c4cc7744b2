// Key pass of the GBLA backward on tensor cores (bf16, D = 64): for every
// valid token t of a (batch, head), with the reduced gradients dS, dz of the
// state and c = <dS, S> + <dz, z> (the chain rule of Sec. 2.1 item 2 through
// the state and the softmax key gate):
//
//   dK^_t = dS v~_t + dz            dk~_t = g_t dK^_t phi'(k~_t)
//   dv~_t = dS^T K^_t               dgate_t = g_t (phi(k~_t) . dK^_t - c)
//
// with K^_t = g_t phi(k~_t), g the softmax gate and phi' = min(phi, 1) (elu + 1:
// phi' = 1 where phi = x + 1 > 1, phi' = e^x = phi where x <= 0).
//
// tc_bwd_key_kernel: persistent, one CTA per SM, each taking a contiguous run
// of 128-token tiles (so the (batch, head) changes rarely).  One TMA warp
// brings the raw k and v rows of a tile (128 tokens + 3 rows of conv history,
// 128B-swizzled) into a 2-deep ring; four producer warps (one token row per
// thread) run both Conv1Ds, phi and the gate in fp32 and write V~ and K^ as
// bf16 K-major A tiles; one thread issues the MMAs
// DK = V~ dS^T and DV = K^ dS (M = 128, N = 64, K = 64) against bf16 hi + lo
// splits of dS, fp32 accumulation in TMEM (two buffers); four epilogue warps
// (one token row per thread) form dk~, dv~ and dgate and write the bf16 dk~ /
// dv~ rows through per-warp staging as whole 128-byte segments.  The epilogue
// warps also build the dS tiles, and add up c from the dS reduction's partial
// sums in order, whenever the (batch, head) changes.
//
// Every mbarrier wait is bounded (2 s); a wait that runs out sets a bit in
// g_bwd_error and the CTA's abort flag, every role leaves its loop, the TMA
// lane waits (bounded) for its copies in flight and the MMA thread for its
// MMAs before TMEM is freed.
#include <math.h>

#include <mutex>

#include "gbla_internal.cuh"
#include "gbla_sm100.cuh"

namespace gbla {

__device__ unsigned int g_bwd_error;

namespace {

using namespace sm100;

constexpr int kD = 64;
constexpr int kKTok = 128;                       // tokens per tile (MMA M)
constexpr int kKRawRows = kKTok + kConvW - 1;    // 131
constexpr int kKRawBox = kKRawRows * 128;        // 16768 bytes per raw box
constexpr int kKRawHalf = (kKRawBox + 1023) / 1024 * 1024;  // 17408
constexpr int kKRawStage = 2 * kKRawHalf;        // k box, v box
constexpr int kKStages = 2;
constexpr int kKTile = kKTok * 128;              // 16384: one 128 x 64 bf16 tile
constexpr int kKAStage = 2 * kKTile;             // V~, K^
constexpr int kKBTile = kD * 128;                // 8192: one 64 x 64 bf16 tile
constexpr int kKProdWarps = 4, kKEpiWarps = 4;
constexpr int kKEpiWarp0 = kKProdWarps;          // 4
constexpr int kKMmaWarp = kKEpiWarp0 + kKEpiWarps;  // 8
constexpr int kKTmaWarp = kKMmaWarp + 1;         // 9
constexpr int kKThreads = (kKTmaWarp + 1) * 32;  // 320
constexpr int kKEpi = kKEpiWarps * 32;
constexpr int kKStg = 32 * 128;                  // staging per epilogue warp: 32 rows x 32 fp32
constexpr uint32_t kKTmemCols = 256;             // two buffers of [DK | DV]

constexpr int kKOffRaw = 0;
constexpr int kKOffA = kKOffRaw + kKStages * kKRawStage;     // 69632
constexpr int kKOffB = kKOffA + kKStages * kKAStage;         // 135168: dS hi, lo, dS^T hi, lo
constexpr int kKOffG = kKOffB + 4 * kKBTile;                 // 167936: float [2][128]
constexpr int kKOffDz = kKOffG + kKStages * kKTok * 4;       // float [64]
constexpr int kKOffStg = kKOffDz + kD * 4;
constexpr int kKOffTaps = kKOffStg + kKEpiWarps * kKStg;     // per producer warp: k, v taps
constexpr int kKTapBytes = 2 * kD * 16;                      // float4 [2][64]
constexpr int kKOffBar = kKOffTaps + kKProdWarps * kKTapBytes;
// raw_full[2], raw_empty[2], a_full[2], a_empty[2], kh_full[2], kh_empty[2],
// acc_full[2], acc_empty[2], b_full, b_free, fin
constexpr int kKBars = 8 * kKStages + 3;
constexpr int kKOffMisc = kKOffBar + kKBars * 8;             // tmem address, abort flag, c
constexpr int kKSmem = kKOffMisc + 16 + 1024;
static_assert(kKSmem <= 227 * 1024, "key-pass shared memory");

struct KeyParams {
  const __nv_bfloat16 *gate;       // [B, N, H]
  const float *conv_w;             // [3, H, D, 4]
  const float2 *stats;             // [B*H]: gate max, sum of exp
  const float *red;                // [B*H][D*D + D]: dS, dz
  const float *dotpart;            // [B*H][ndot]: partials of c = <dS, S> + <dz, z>
  int ndot;
  const int32_t *seq_lens;
  __nv_bfloat16 *dkt, *dvt;        // [B, N, H, D] bf16 planes
  __nv_bfloat16 *dgate;            // [B, N, H]
  int B, H, N, tps;
};

__device__ __forceinline__ void report(unsigned code, const AbortFlag &ab) {
  atomicOr(&g_bwd_error, code);
  ab.raise();
}



__device__ __forceinline__ int seq_len(const int32_t *seq_lens, int b, int N) {
  if (seq_lens == nullptr) return N;
  const int L = seq_lens[b];
  return L < 0 ? 0 : (L > N ? N : L);
}

// Tile i of this CTA's contiguous run -> (b, h, t0, L); false for a tile that
// lies wholly in the padding.
struct KTile {
  int bh, b, h, t0, L;
};
__device__ __forceinline__ bool key_tile(const KeyParams &p, int i, KTile &t) {
  t.bh = i / p.tps;
  t.b = t.bh / p.H;
  t.h = t.bh % p.H;
  t.t0 = (i - t.bh * p.tps) * kKTok;
  t.L = seq_len(p.seq_lens, t.b, p.N);
  return t.t0 < t.L;
}

__device__ __forceinline__ void unpack8(uint4 r, float (&f)[8]) {
  const float2 a = bf2_to_f2(r.x), b = bf2_to_f2(r.y), c = bf2_to_f2(r.z), d = bf2_to_f2(r.w);
  f[0] = a.x; f[1] = a.y; f[2] = b.x; f[3] = b.y;
  f[4] = c.x; f[5] = c.y; f[6] = d.x; f[7] = d.y;
}
__device__ __forceinline__ uint4 pack8(const float (&f)[8]) {
  return make_uint4(f2_to_bf2(f[0], f[1]), f2_to_bf2(f[2], f[3]), f2_to_bf2(f[4], f[5]),
                    f2_to_bf2(f[6], f[7]));
}
// byte offset of 16-byte chunk c of row r in a 128B-swizzled K-major tile
__device__ __forceinline__ uint32_t sw_off(int r, int c) {
  return (uint32_t)((r >> 3) * 1024 + (r & 7) * 128 + ((c ^ (r & 7)) << 4));
}
// n consecutive fp32 values (16-byte aligned) from shared memory, 16 bytes per
// load; every lane reads the same address (a broadcast)
template <int n>
__device__ __forceinline__ void lds_f32n(uint32_t a, float (&f)[n]) {
#pragma unroll
  for (int k = 0; k < n / 4; ++k) {
    const uint4 u = lds_v4(a + 16 * k);
    f[4 * k] = __uint_as_float(u.x);
    f[4 * k + 1] = __uint_as_float(u.y);
    f[4 * k + 2] = __uint_as_float(u.z);
    f[4 * k + 3] = __uint_as_float(u.w);
  }
}
// phi = elu + 1, branch-free: the exponential of min(x, 0) is always taken and
// then selected (measured 7 % faster per backward step than a branch around
// expf, which in turn beat a branch around __expf).
__device__ __forceinline__ float phi_f(float x) {
  const float ex = exp2f(fminf(x, 0.f) * 1.4426950408889634f);
  return x > 0.f ? x + 1.f : ex;
}

__global__ void __launch_bounds__(kKThreads, 1)
    tc_bwd_key_kernel(const KeyParams p, const __grid_constant__ CUtensorMap tm_k,
                      const __grid_constant__ CUtensorMap tm_v) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int H = p.H, N = p.N;

  uint64_t *bars = (uint64_t *)(smem + kKOffBar);
  uint64_t *raw_full = bars, *raw_empty = bars + 2, *a_full = bars + 4, *a_empty = bars + 6;
  // kh_full / kh_empty: the epilogue's reads of the K^ rows of an A stage
  uint64_t *kh_full = bars + 8, *kh_empty = bars + 10, *acc_full = bars + 12;
  uint64_t *acc_empty = bars + 14, *b_full = bars + 16, *b_free = bars + 17, *fin = bars + 18;
  uint32_t *tmem_slot = (uint32_t *)(smem + kKOffMisc);
  const AbortFlag ab{smem_u32(smem + kKOffMisc + 4)};
  float *cslot = (float *)(smem + kKOffMisc + 8);

  const long long T = (long long)p.B * H * p.tps;
  // tile indices fit an int (checked on the host)
  const int i0 = (int)(T * blockIdx.x / gridDim.x), i1 = (int)(T * (blockIdx.x + 1) / gridDim.x);
  if (i0 >= i1) return;

  if (tid == 0) {
    for (int i = 0; i < kKStages; ++i) {
      mbar_init(&raw_full[i], 1);
      mbar_init(&raw_empty[i], kKProdWarps);
      mbar_init(&a_full[i], kKProdWarps);
      mbar_init(&a_empty[i], 1);
      mbar_init(&kh_full[i], kKProdWarps);
      mbar_init(&kh_empty[i], kKEpiWarps);
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], kKEpiWarps);
    }
    mbar_init(b_full, 1);
    mbar_init(b_free, 1);
    mbar_init(fin, 1);
    *(volatile int *)(smem + kKOffMisc + 4) = 0;
    fence_mbar_init();
  }
  if (warp == kKTmaWarp && lane == 0) {
    tma_prefetch_desc(&tm_k);
    tma_prefetch_desc(&tm_v);
  }
  if (warp == kKMmaWarp) tmem_alloc(tmem_slot, kKTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // launched with programmatic dependent launch: dS, dz and the partials of c
  // come from the reduction before, and nothing global is written before it
  // has completed
  grid_dep_wait();
  grid_dep_launch();

  if (warp == kKTmaWarp) {
    // ------------------------------------------------------------ TMA: raw k, v rows
    if (lane == 0) {
      int li = 0;
      bool ok = true;
      for (int i = i0; i < i1 && ok; ++i) {
        KTile t;
        if (!key_tile(p, i, t)) continue;
        const int s = li % kKStages;
        if (!mbar_wait(&raw_empty[s], ((li / kKStages) & 1) ^ 1, &ab)) {
          if (!ab.raised()) report(1, ab);
          ok = false;
          break;
        }
        uint8_t *dst = smem + kKOffRaw + s * kKRawStage;
        mbar_arrive_expect_tx(&raw_full[s], 2 * kKRawBox);
        // rows t0 - 3 .. t0 + 127; rows before the sequence start read as zeros
        tma_load_4d(dst, &tm_k, &raw_full[s], 0, t.h, t.t0 - 3, t.b);
        tma_load_4d(dst + kKRawHalf, &tm_v, &raw_full[s], 0, t.h, t.t0 - 3, t.b);
        ++li;
      }
      for (int j = li - 1; j >= 0 && j >= li - kKStages; --j)
        if (!mbar_wait(&raw_full[j % kKStages], (j / kKStages) & 1, nullptr)) report(2, ab);
    }
  } else if (warp < kKEpiWarp0) {
    // ------------------------------------------------------------ producers
    const int r = tid;  // tile row
    // this warp's own copy of the head's k and v taps (rewritten when the
    // (b, h) changes; a warp only reads the copy it wrote, so __syncwarp orders it)
    const uint32_t taps = smem_u32(smem + kKOffTaps + warp * kKTapBytes);
    // The gate value and the head's softmax statistics of the NEXT tile are
    // loaded one tile ahead, so their global-load latency hides behind this
    // tile's Conv1D work (the producers are the slowest role of the pass).
    auto next_tile = [&](int j, KTile &tn) {
      for (; j < i1; ++j)
        if (key_tile(p, j, tn)) return j;
      return i1;
    };
    auto gate_raw = [&](const KTile &tn) {
      const int tok = tn.t0 + r;
      return tok < tn.L ? p.gate[((size_t)tn.b * N + tok) * H + tn.h] : __float2bfloat16_rn(0.f);
    };
    int li = 0, cur_bh = -1;
    bool ok = true;
    KTile t;
    int i = next_tile(i0, t);
    __nv_bfloat16 graw = i < i1 ? gate_raw(t) : __float2bfloat16_rn(0.f);
    float2 gs = i < i1 ? p.stats[t.bh] : make_float2(0.f, 1.f);
    while (i < i1 && ok) {
      KTile tn;
      const int inext = next_tile(i + 1, tn);
      __nv_bfloat16 graw_n = __float2bfloat16_rn(0.f);
      float2 gs_n = gs;
      if (inext < i1) {
        graw_n = gate_raw(tn);
        if (tn.bh != t.bh) gs_n = p.stats[tn.bh];
      }
      const int s = li % kKStages;
      if (t.bh != cur_bh) {
        cur_bh = t.bh;
        __syncwarp();  // the previous head's taps are no longer read
        for (int u = lane; u < 2 * kD; u += 32) {
          const int str = 1 + u / kD, ch = u % kD;  // stream 1 (k) or 2 (v)
          const float4 t4 = __ldg((const float4 *)(p.conv_w + ((size_t)(str * H + t.h) * kD + ch) * kConvW));
          *(float4 *)(smem + kKOffTaps + warp * kKTapBytes + 16 * u) = t4;
        }
        __syncwarp();
      }
      const int tok = t.t0 + r;
      const bool valid = tok < t.L;
      const float g = valid ? expf(__bfloat162float(graw) - gs.x) / gs.y : 0.f;
      const bool w = mbar_wait(&raw_full[s], (li / kKStages) & 1, &ab) &&
                     mbar_wait(&a_empty[s], ((li / kKStages) & 1) ^ 1, &ab) &&
                     mbar_wait(&kh_empty[s], ((li / kKStages) & 1) ^ 1, &ab);
      if (!__all_sync(0xffffffffu, w)) {  // the whole warp leaves together
        ok = false;
        break;
      }
      const uint32_t rk = smem_u32(smem + kKOffRaw + s * kKRawStage);
      const uint32_t rv = rk + kKRawHalf;
      const uint32_t av = smem_u32(smem + kKOffA + s * kKAStage);
      const uint32_t ak = av + kKTile;
#pragma unroll 2
      for (int c = 0; c < kD / 8; ++c) {
        float kx[kConvW][8], vx[kConvW][8];
#pragma unroll
        for (int j = 0; j < kConvW; ++j) {
          unpack8(lds_v4(rk + sw_off(r + j, c)), kx[j]);
          unpack8(lds_v4(rv + sw_off(r + j, c)), vx[j]);
        }
        float vt[8], kh[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const uint4 uk = lds_v4(taps + 16 * (8 * c + e));
          const uint4 uv = lds_v4(taps + 16 * (kD + 8 * c + e));
          const float4 tk = make_float4(__uint_as_float(uk.x), __uint_as_float(uk.y),
                                        __uint_as_float(uk.z), __uint_as_float(uk.w));
          const float4 tv = make_float4(__uint_as_float(uv.x), __uint_as_float(uv.y),
                                        __uint_as_float(uv.z), __uint_as_float(uv.w));
          const float kt = fmaf(tk.w, kx[3][e], fmaf(tk.z, kx[2][e], fmaf(tk.y, kx[1][e], tk.x * kx[0][e])));
          const float v1 = fmaf(tv.w, vx[3][e], fmaf(tv.z, vx[2][e], fmaf(tv.y, vx[1][e], tv.x * vx[0][e])));
          vt[e] = valid ? v1 : 0.f;
          kh[e] = g * phi_f(kt);  // 0 on padded rows (g = 0)
        }
        const uint32_t o = sw_off(r, c);
        sts_v4(av + o, pack8(vt));
        sts_v4(ak + o, pack8(kh));
      }
      sts_f32(smem_u32(smem + kKOffG) + (uint32_t)(s * kKTok + r) * 4, g);
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&raw_empty[s]);
        mbar_arrive(&a_full[s]);
        mbar_arrive(&kh_full[s]);
      }
      ++li;
      i = inext;
      t = tn;
      graw = graw_n;
      gs = gs_n;
    }
    if (!ok && !ab.raised()) report(4, ab);
  } else if (warp < kKMmaWarp) {
    // ------------------------------------------------------------ epilogue
    const int q4 = warp & 3, row = 32 * q4 + lane;
    const int et = tid - kKEpiWarp0 * 32;  // 0..127
    const uint32_t stg = smem_u32(smem + kKOffStg + (warp - kKEpiWarp0) * kKStg);
    const uint32_t bb = smem_u32(smem + kKOffB);
    const uint32_t dzs = smem_u32(smem + kKOffDz);
    // Every epilogue warp runs every iteration (a failed wait does not leave
    // the loop), so the named barriers below always match.
    int li = 0, cur_bh = -1, nbh = 0;
    bool ok = true;
    for (int i = i0; i < i1; ++i) {
      KTile t;
      if (!key_tile(p, i, t)) continue;
      const int s = li % kKStages, buf = li % 2;
      if (t.bh != cur_bh) {
        // dS of the new (b, h) as bf16 hi + lo: dS (rows d, K = e) for DK and
        // dS^T (rows e, K = d) for DV, once the previous MMAs are done with them
        if (nbh > 0) {
          named_barrier(1, kKEpi);  // every epilogue warp is done with the previous tile
          ok = mbar_wait(b_free, (nbh - 1) & 1, &ab) && ok;
        }
        const float *dS = p.red + (size_t)t.bh * (kD * kD + kD);
        for (int u = et; u < kD * (kD / 8); u += kKEpi) {
          const int rr = u >> 3, cc = u & 7;  // row rr, chunk cc
          float hi[8], lo[8], hT[8], lT[8];
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const float x = dS[rr * kD + 8 * cc + e];           // dS[rr][8cc + e]
            const float y = dS[(8 * cc + e) * kD + rr];         // dS^T[rr][8cc + e]
            hi[e] = __bfloat162float(__float2bfloat16_rn(x));
            lo[e] = x - hi[e];
            hT[e] = __bfloat162float(__float2bfloat16_rn(y));
            lT[e] = y - hT[e];
          }
          const uint32_t o = sw_off(rr, cc);
          sts_v4(bb + o, pack8(hi));
          sts_v4(bb + kKBTile + o, pack8(lo));
          sts_v4(bb + 2 * kKBTile + o, pack8(hT));
          sts_v4(bb + 3 * kKBTile + o, pack8(lT));
        }
        if (et < kD) ((float *)(smem + kKOffDz))[et] = dS[kD * kD + et];
        if (et == 0) {  // c, the partials added in order
          float c = 0.f;
          for (int j = 0; j < p.ndot; ++j) c += p.dotpart[(size_t)t.bh * p.ndot + j];
          *cslot = c;
        }
        fence_proxy_async_smem();
        named_barrier(1, kKEpi);
        if (et == 0) mbar_arrive(b_full);
        cur_bh = t.bh;
        ++nbh;
      }
      ok = mbar_wait(&acc_full[buf], (li >> 1) & 1, &ab) && ok;
      ok = mbar_wait(&kh_full[s], (li / kKStages) & 1, &ab) && ok;
      tc_fence_after();
      const uint32_t tacc = tmem + ((uint32_t)(32 * q4) << 16) + buf * 128;
      const int tok = t.t0 + row;
      const bool valid = tok < t.L;
      const float g = lds_f32(smem_u32(smem + kKOffG) + (uint32_t)(s * kKTok + row) * 4);
      // K^ = g phi(k~) (the MMA's bf16 A tile) stands in for phi(k~):
      //   dk~ = g dK^ min(phi, 1) = dK^ min(K^, g),
      //   dgate = g (phi . dK^ - c) = K^ . dK^ - g c
      const uint32_t ak = smem_u32(smem + kKOffA + s * kKAStage) + kKTile;
      const size_t prow = (((size_t)t.b * N + t.t0) * H + t.h) * kD;  // plane row of tile row 0
      const size_t prs = (size_t)H * kD;                               // plane row stride
      float khdk = 0.f;
      // dk~ in two 32-column halves, then dv~; each row of 64 bf16 goes through
      // the staging rows as one 128-byte segment
#pragma unroll 1
      for (int mat = 0; mat < 2; ++mat) {  // dk~, then dv~
        uint4 pk[8];
#pragma unroll
        for (int hp = 0; hp < 2; ++hp) {  // 32-column halves
          const int part = 2 * mat + hp;
          float v[32];
          tmem_ld16(tacc + 32 * part, *reinterpret_cast<float(*)[16]>(v));
          tmem_ld16(tacc + 32 * part + 16, *reinterpret_cast<float(*)[16]>(v + 16));
          tmem_ld_wait();
          if (part == 3) {  // accumulators drained
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&acc_empty[buf]);
          }
          if (mat == 0) {
#pragma unroll
            for (int cq = 0; cq < 4; ++cq) {
              float kh[8], dz8[8];
              unpack8(lds_v4(ak + sw_off(row, 4 * hp + cq)), kh);
              lds_f32n(dzs + 4 * (32 * hp + 8 * cq), dz8);
#pragma unroll
              for (int e = 0; e < 8; ++e) {
                const float dk = v[8 * cq + e] + dz8[e];
                khdk = fmaf(kh[e], dk, khdk);
                v[8 * cq + e] = dk * fminf(kh[e], g);
              }
            }
            if (hp == 1) {
              __syncwarp();
              if (lane == 0) mbar_arrive(&kh_empty[s]);  // K^ rows read
            }
          }
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            float a[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) a[e] = v[8 * j + e];
            pk[4 * hp + j] = pack8(a);
          }
        }
#pragma unroll
        for (int j = 0; j < 8; ++j) sts_v4(stg + lane * 128 + ((j ^ (lane & 7)) << 4), pk[j]);
        __syncwarp();
        __nv_bfloat16 *plane = mat == 0 ? p.dkt : p.dvt;
#pragma unroll
        for (int it = 0; it < 8; ++it) {
          const int rr = it * 4 + (lane >> 3), ch = lane & 7;
          const uint4 val = lds_v4(stg + rr * 128 + ((ch ^ (rr & 7)) << 4));
          const int trow = 32 * q4 + rr;
          if (t.t0 + trow < t.L) *(uint4 *)(plane + prow + (size_t)trow * prs + ch * 8) = val;
        }
        __syncwarp();
      }
      if (valid)
        p.dgate[((size_t)t.b * N + tok) * H + t.h] = __float2bfloat16_rn(khdk - g * *cslot);
      ++li;
    }
    if (!ok && !ab.raised()) report(8, ab);
  } else if (warp == kKMmaWarp) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16_f32(kKTok, kD, 0, 0);
      const uint32_t bb = smem_u32(smem + kKOffB);
      int li = 0, cur_bh = -1, nbh = 0;
      bool ok = true;
      for (int i = i0; i < i1 && ok; ++i) {
        KTile t;
        if (!key_tile(p, i, t)) continue;
        const int s = li % kKStages, buf = li % 2;
        if (t.bh != cur_bh) {
          if (!mbar_wait(b_full, nbh & 1, &ab)) {
            ok = false;
            break;
          }
          cur_bh = t.bh;
          ++nbh;
        }
        if (!mbar_wait(&a_full[s], (li / kKStages) & 1, &ab) ||
            !mbar_wait(&acc_empty[buf], ((li >> 1) & 1) ^ 1, &ab)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t av = smem_u32(smem + kKOffA + s * kKAStage), ak = av + kKTile;
        const uint32_t dk = tmem + buf * 128, dv = dk + kD;
#pragma unroll
        for (int k16 = 0; k16 < 4; ++k16) {
          const uint32_t ko = 32 * k16;
          const uint64_t a1 = sw128_desc(av + ko, 16, 1024), a2 = sw128_desc(ak + ko, 16, 1024);
          mma_bf16(dk, a1, sw128_desc(bb + ko, 16, 1024), idesc, k16 != 0);
          mma_bf16(dk, a1, sw128_desc(bb + kKBTile + ko, 16, 1024), idesc, 1);
          mma_bf16(dv, a2, sw128_desc(bb + 2 * kKBTile + ko, 16, 1024), idesc, k16 != 0);
          mma_bf16(dv, a2, sw128_desc(bb + 3 * kKBTile + ko, 16, 1024), idesc, 1);
        }
        mma_commit(&a_empty[s]);
        mma_commit(&acc_full[buf]);
        // last tile of this (b, h) in this CTA: the dS tiles may be rebuilt
        bool last = true;
        for (int j = i + 1; j < i1; ++j) {
          KTile tn;
          if (key_tile(p, j, tn)) {
            last = tn.bh != t.bh;
            break;
          }
        }
        if (last) mma_commit(b_free);
        ++li;
      }
      if (!ok && !ab.raised()) report(16, ab);
      mma_commit(fin);
      if (!mbar_wait(fin, 0, nullptr)) report(32, ab);
    }
  }
  __syncthreads();
  if (warp == kKMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem, kKTmemCols);
  }
}

// ===================================================================== query pass
// Per (b, h, chunk of 1024 tokens), for every valid token t with P_t = phi(q~_t),
// the forward's O_t = S^T P_t / (P_t . z) and the gated RMSNorm (Sec. 2.1
// items 2 and 3), the chain rule in reverse:
//
//   dog_t = dy O r w silu'(og);  dnw += dy O r silu(og);  u = dy w silu(og)
//   dO = r u - (r^3 / D) O (u . O);  dnum = dO / den;  dden = -(dO . O) / den
//   dq~_t = (S dnum_t + z dden_t) phi'(q~_t);  dS += P_t dnum_t^T;  dz += P_t dden_t
//
// Four MMAs per 128-token tile: [num | den] = P [S | z] (S as bf16 hi + lo);
// dP = dnum S^T (hi + lo); dS += P^T dnum (both operands read MN-major from the
// same tiles, M = 128 with the two 64-row halves of A equal, accumulated in
// TMEM over the chunk).  Roles: a TMA warp (raw q tile with 3 rows of history,
// out_gate and dy tiles), four producer warps (P = phi(conv(q)) in fp32, bf16
// A tile), one MMA thread, and two groups of four warps taking the even and
// the odd tiles (one token row per thread: the gated-RMSNorm / readout
// backward, then dq~; per-warp dnw and dz sums); the chunk's dS, dz and dnw
// go to a partial record.  One CTA per (b, h, chunk); the chunk length is
// chosen on the host so that the chunks of all (b, h) fit one wave of CTAs
// where they can (each CTA pays the pipeline fill once).
constexpr int kQInQ = kKRawHalf;                   // 17408: raw q box
constexpr int kQIn = kQInQ + 2 * kKTile;           // + out_gate, dy tiles: 50176
constexpr int kQSzT = 80 * 128;                    // [S^T | z] tile: 80 rows
constexpr int kQProdWarps = 4, kQE1Warps = 4, kQE2Warps = 4;
constexpr int kQE1Warp0 = kQProdWarps;             // 4
constexpr int kQE2Warp0 = kQE1Warp0 + kQE1Warps;   // 8
constexpr int kQMmaWarp = kQE2Warp0 + kQE2Warps;   // 12
constexpr int kQTmaWarp = kQMmaWarp + 1;           // 13
constexpr int kQThreads = (kQTmaWarp + 1) * 32;    // 448
constexpr int kQOffIn = 0;
constexpr int kQOffP = kQOffIn + kKStages * kQIn;          // 100352
constexpr int kQOffDn = kQOffP + kKStages * kKTile;        // 133120
constexpr int kQOffB = kQOffDn + kKStages * kKTile;        // 165888: SzT hi, lo, S hi, lo
constexpr int kQOffZ = kQOffB + 2 * kQSzT + 2 * kKBTile;   // 202752: z [64], w [64]
constexpr int kQOffTaps = kQOffZ + 2 * kD * 4;             // float4 [64]: q taps of the head
constexpr int kQOffBar = kQOffTaps + kD * 16;
// in_full, in_empty, p_full, p_empty, a1_full, a1_empty, dn_full, dn_empty,
// a2_full, a2_empty (2 each), b_full, a3_full, fin
constexpr int kQBars = 10 * kKStages + 3;
constexpr int kQOffMisc = kQOffBar + kQBars * 8;
constexpr int kQSmem = kQOffMisc + 16 + 1024;
static_assert(kQSmem <= 227 * 1024, "query-pass shared memory");
static_assert(16 * kD * 4 <= kKStages * kQIn, "end-of-chunk reduction space");
constexpr uint32_t kQA1 = 0, kQA2 = 256, kQA3 = 384;     // TMEM columns
constexpr int kQRec = kD * kD + 2 * kD;            // dS, dz, dnw

struct QueryParams {
  const float *conv_w, *norm_w, *state;  // state: [B*H][D*D + D]
  const int32_t *seq_lens;
  __nv_bfloat16 *dog;                    // [B, N, H, D]
  __nv_bfloat16 *dqt;                    // bf16 plane
  float *part;                           // [B*H][nck][kQRec]
  float eps;
  int B, H, N, nck;
  int ctiles;  // 128-token tiles per chunk
};

// sigmoid(x) = (1 + tanh(x / 2)) / 2 with the hardware tanh approximation (an
// absolute error below 2^-11, inside the bf16 tolerance): one special-function
// operation instead of an exponential and a reciprocal.
__device__ __forceinline__ float sigmoid_f(float x) {
  float y;
  asm("tanh.approx.f32 %0, %1;" : "=f"(y) : "f"(0.5f * x));
  return fmaf(0.5f, y, 0.5f);
}

// Column sums over the 32 rows of a warp (one row per lane) of n = 16 or 32
// columns held one row per lane in x: recursive halving with shuffles, in a
// fixed order.  n = 32: lane l returns the sum of column l; n = 16: lanes l
// and l ^ 1 both return the sum of column l >> 1.  x is overwritten.
template <int n>
__device__ __forceinline__ float lane_colsum(float (&x)[n]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int o = 16, m = n; o > 0 && m > 1; o >>= 1, m >>= 1) {
    const bool up = lane & o;
#pragma unroll
    for (int i = 0; i < m / 2; ++i) {
      const float keep = up ? x[i + m / 2] : x[i];
      const float send = up ? x[i] : x[i + m / 2];
      x[i] = keep + __shfl_xor_sync(0xffffffffu, send, o);
    }
  }
  if (n == 16) x[0] += __shfl_xor_sync(0xffffffffu, x[0], 1);
  return x[0];
}

__global__ void __launch_bounds__(kQThreads, 1)
    tc_bwd_query_kernel(const QueryParams p, const __grid_constant__ CUtensorMap tm_q,
                        const __grid_constant__ CUtensorMap tm_og,
                        const __grid_constant__ CUtensorMap tm_dy) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int H = p.H, N = p.N;
  const int chunk = blockIdx.x, bh = blockIdx.y, b = bh / H, h = bh % H;
  const int L = seq_len(p.seq_lens, b, N);
  const int c0 = chunk * p.ctiles * kKTok;
  // valid tiles of this chunk: t0 = c0 + 128 j < min(L, N)
  const int nt = L > c0 ? min(p.ctiles, (L - c0 + kKTok - 1) / kKTok) : 0;

  uint64_t *bars = (uint64_t *)(smem + kQOffBar);
  uint64_t *in_full = bars, *in_empty = bars + 2, *p_full = bars + 4, *p_empty = bars + 6;
  uint64_t *a1_full = bars + 8, *a1_empty = bars + 10, *dn_full = bars + 12;
  uint64_t *dn_empty = bars + 14, *a2_full = bars + 16, *a2_empty = bars + 18;
  uint64_t *b_full = bars + 20, *a3_full = bars + 21, *fin = bars + 22;
  uint32_t *tmem_slot = (uint32_t *)(smem + kQOffMisc);
  const AbortFlag ab{smem_u32(smem + kQOffMisc + 4)};
  const uint32_t zs = smem_u32(smem + kQOffZ), ws = zs + 4 * kD;  // z [64], norm w [64]

  if (tid == 0) {
    for (int i = 0; i < kKStages; ++i) {
      mbar_init(&in_full[i], 1);
      mbar_init(&in_empty[i], kQProdWarps + kQE1Warps);
      mbar_init(&p_full[i], kQProdWarps);
      mbar_init(&p_empty[i], 1 + kQE2Warps);
      mbar_init(&a1_full[i], 1);
      mbar_init(&a1_empty[i], kQE1Warps);
      mbar_init(&dn_full[i], kQE1Warps);
      mbar_init(&dn_empty[i], 1);
      mbar_init(&a2_full[i], 1);
      mbar_init(&a2_empty[i], kQE2Warps);
    }
    mbar_init(b_full, 1);
    mbar_init(a3_full, 1);
    mbar_init(fin, 1);
    *(volatile int *)(smem + kQOffMisc + 4) = 0;
    fence_mbar_init();
  }
  if (tid < kD)  // the head's q taps, read by the producers
    *(float4 *)(smem + kQOffTaps + 16 * tid) =
        __ldg((const float4 *)(p.conv_w + ((size_t)h * kD + tid) * kConvW));
  // launched with programmatic dependent launch: the state may come from the
  // kernel before, and nothing global is written before it has completed
  grid_dep_wait();
  grid_dep_launch();
  {
    // B tiles from S (every thread; contiguous 32-byte reads of S rows, all in
    // flight together): S as bf16 hi + lo with rows d, K = e (for dP), and its
    // transpose [S^T | z] with rows e, K = d, row 64 = z, rows 65..79 zero (for
    // [num | den]); K-major, 128B-swizzled.
    const float *S = p.state + (size_t)bh * (kD * kD + kD);
    const uint32_t bb = smem_u32(smem + kQOffB);
    uint8_t *bsz = smem + kQOffB;
    for (int u = tid; u < kD * (kD / 8); u += kQThreads) {
      const int rr = u >> 3, cc = u & 7;  // S row rr, columns 8 cc ..
      const float4 x0 = __ldg((const float4 *)(S + rr * kD + 8 * cc));
      const float4 x1 = __ldg((const float4 *)(S + rr * kD + 8 * cc + 4));
      const float x[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
      float hi[8], lo[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        hi[e] = __bfloat162float(__float2bfloat16_rn(x[e]));
        lo[e] = x[e] - hi[e];
      }
      sts_v4(bb + 2 * kQSzT + sw_off(rr, cc), pack8(hi));
      sts_v4(bb + 2 * kQSzT + kKBTile + sw_off(rr, cc), pack8(lo));
      // transposed: element (row e = 8 cc + i, K = rr)
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const uint32_t o = sw_off(8 * cc + i, rr >> 3) + (rr & 7) * 2;
        *(__nv_bfloat16 *)(bsz + o) = __float2bfloat16_rn(hi[i]);
        *(__nv_bfloat16 *)(bsz + kQSzT + o) = __float2bfloat16_rn(lo[i]);
      }
    }
    for (int u = tid; u < 16 * (kD / 8); u += kQThreads) {  // rows 64 (z) .. 79
      const int rr = kD + (u >> 3), cc = u & 7;
      float hi[8], lo[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        const float x = rr == kD ? S[kD * kD + 8 * cc + e] : 0.f;
        hi[e] = __bfloat162float(__float2bfloat16_rn(x));
        lo[e] = x - hi[e];
      }
      sts_v4(bb + sw_off(rr, cc), pack8(hi));
      sts_v4(bb + kQSzT + sw_off(rr, cc), pack8(lo));
    }
    if (tid < kD) {
      ((float *)(smem + kQOffZ))[tid] = S[kD * kD + tid];
      ((float *)(smem + kQOffZ))[kD + tid] = p.norm_w[(size_t)h * kD + tid];
    }
    fence_proxy_async_smem();
  }
  if (warp == kQTmaWarp && lane == 0) {
    tma_prefetch_desc(&tm_q);
    tma_prefetch_desc(&tm_og);
    tma_prefetch_desc(&tm_dy);
  }
  if (warp == kQMmaWarp) tmem_alloc(tmem_slot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const size_t prs = (size_t)H * kD;                         // plane row stride
  const size_t prow0 = (((size_t)b * N + c0) * H + h) * kD;  // plane row of the chunk's token 0
  // column sums of the epilogue groups (kept until every role is done):
  // dnorm_w column 16 j + (lane >> 1) and dz column 32 part + lane of a warp's rows
  float dnw4[4] = {0.f, 0.f, 0.f, 0.f};
  float dz2[2] = {0.f, 0.f};

  if (warp == kQTmaWarp) {
    // ------------------------------------------------------------ TMA: q, out_gate, dy
    if (lane == 0) {
      int li = 0;
      for (; li < nt; ++li) {
        const int s = li % kKStages, t0 = c0 + li * kKTok;
        if (!mbar_wait(&in_empty[s], ((li / kKStages) & 1) ^ 1, &ab)) {
          if (!ab.raised()) report(64, ab);
          break;
        }
        uint8_t *dst = smem + kQOffIn + s * kQIn;
        mbar_arrive_expect_tx(&in_full[s], kKRawBox + 2 * kKTile);
        tma_load_4d(dst, &tm_q, &in_full[s], 0, h, t0 - 3, b);
        tma_load_4d(dst + kQInQ, &tm_og, &in_full[s], 0, h, t0, b);
        tma_load_4d(dst + kQInQ + kKTile, &tm_dy, &in_full[s], 0, h, t0, b);
      }
      for (int j = li - 1; j >= 0 && j >= li - kKStages; --j)
        if (!mbar_wait(&in_full[j % kKStages], (j / kKStages) & 1, nullptr)) report(128, ab);
    }
  } else if (warp < kQE1Warp0) {
    // ------------------------------------------------------------ producers: P = phi(conv(q))
    const int r = tid;
    const uint32_t taps = smem_u32(smem + kQOffTaps);
    bool ok = true;
    for (int li = 0; li < nt && ok; ++li) {
      const int s = li % kKStages, ph = (li / kKStages) & 1;
      const bool valid = c0 + li * kKTok + r < L;
      const bool w = mbar_wait(&in_full[s], ph, &ab) && mbar_wait(&p_empty[s], ph ^ 1, &ab);
      if (!__all_sync(0xffffffffu, w)) {  // the whole warp leaves together
        ok = false;
        break;
      }
      const uint32_t rq = smem_u32(smem + kQOffIn + s * kQIn);
      const uint32_t pt = smem_u32(smem + kQOffP + s * kKTile);
#pragma unroll 2
      for (int c = 0; c < kD / 8; ++c) {
        float qx[kConvW][8], pv[8];
#pragma unroll
        for (int j = 0; j < kConvW; ++j) unpack8(lds_v4(rq + sw_off(r + j, c)), qx[j]);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const uint4 tu = lds_v4(taps + 16 * (8 * c + e));
          const float4 tq = make_float4(__uint_as_float(tu.x), __uint_as_float(tu.y),
                                        __uint_as_float(tu.z), __uint_as_float(tu.w));
          const float qt = fmaf(tq.w, qx[3][e], fmaf(tq.z, qx[2][e], fmaf(tq.y, qx[1][e], tq.x * qx[0][e])));
          pv[e] = valid ? phi_f(qt) : 0.f;
        }
        sts_v4(pt + sw_off(r, c), pack8(pv));
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&p_full[s]);
        mbar_arrive(&in_empty[s]);
      }
    }
    if (!ok && !ab.raised()) report(256, ab);
  } else if (warp < kQMmaWarp) {
    // ------------------------------------------------------------ epilogue groups
    // Two groups of four warps (one per TMEM lane quarter, one token row per
    // thread) take the even and the odd tiles: for each, the gated-RMSNorm /
    // readout backward (dog, dnum, dden, dnorm_w sums), then, once the dP / dS
    // MMAs are done, dq~ and the dz sums.  The groups overlap one another.
    const int grp = (warp - kQE1Warp0) >> 2;
    const int q4 = warp & 3, row = 32 * q4 + lane;
    bool ok = true;
    for (int li = grp; li < nt && ok; li += 2) {
      const int s = li % kKStages, ph = (li / kKStages) & 1;
      const int t = c0 + li * kKTok + row;
      const bool valid = t < L;
      const bool w = mbar_wait(&a1_full[s], ph, &ab) && mbar_wait(&in_full[s], ph, &ab) &&
                     mbar_wait(&dn_empty[s], ph ^ 1, &ab);
      if (!__all_sync(0xffffffffu, w)) {  // the whole warp leaves together
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t ta = tmem + ((uint32_t)(32 * q4) << 16) + kQA1 + 128 * s;
      const uint32_t ogt = smem_u32(smem + kQOffIn + s * kQIn) + kQInQ, dyt = ogt + kKTile;
      const uint32_t dnt = smem_u32(smem + kQOffDn + s * kKTile);
      float den;
      {
        float v4[4];
        tmem_ld4(ta + kD, v4);
        tmem_ld_wait();
        den = v4[0];
      }
      const float inv = valid ? 1.f / den : 0.f;
      // pass 1 (nothing here needs r): sum O^2, u . O with u = dy w silu(og) (both
      // summed over the accumulator num = O den and scaled once by 1/den), and
      // two per-element factors that replace this row's out_gate and dy values
      // (read only by this thread from here on): A = dy w silu'(og) (dog = A O r)
      // and Bv = dy silu(og) (dnorm_w term Bv O r, u = Bv w)
      float ss = 0.f, uo = 0.f;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        float v[16], og[16], dy[16];
        tmem_ld16(ta + 16 * j, v);
        unpack8(lds_v4(ogt + sw_off(row, 2 * j)), *reinterpret_cast<float(*)[8]>(og));
        unpack8(lds_v4(ogt + sw_off(row, 2 * j + 1)), *reinterpret_cast<float(*)[8]>(og + 8));
        unpack8(lds_v4(dyt + sw_off(row, 2 * j)), *reinterpret_cast<float(*)[8]>(dy));
        unpack8(lds_v4(dyt + sw_off(row, 2 * j + 1)), *reinterpret_cast<float(*)[8]>(dy + 8));
        float wv[16];
        lds_f32n(ws + 64 * j, wv);
        tmem_ld_wait_regs(v);
        float fa[16], fb[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const float sg = sigmoid_f(og[i]), si = og[i] * sg;
          const float w = wv[i];
          ss = fmaf(v[i], v[i], ss);
          uo = fmaf(dy[i] * w * si, v[i], uo);
          fa[i] = dy[i] * w * sg * (1.f + og[i] * (1.f - sg));
          fb[i] = dy[i] * si;
        }
        float a[8], c[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          a[i] = fa[i];
          c[i] = fa[8 + i];
        }
        sts_v4(ogt + sw_off(row, 2 * j), pack8(a));
        sts_v4(ogt + sw_off(row, 2 * j + 1), pack8(c));
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          a[i] = fb[i];
          c[i] = fb[8 + i];
        }
        sts_v4(dyt + sw_off(row, 2 * j), pack8(a));
        sts_v4(dyt + sw_off(row, 2 * j + 1), pack8(c));
      }
      ss *= inv * inv;
      uo *= inv;
      const float rr = rsqrtf(ss * (1.f / kD) + p.eps);
      const float r3 = rr * rr * rr * (1.f / kD);
      // pass 2: dog, dnorm_w, dnum (bf16 A / B tile); dO . O in closed form:
      // sum_d (r u_d - r3 O_d (u . O)) O_d = r (u . O) - r3 (u . O) sum O^2
      const float doo = rr * uo - r3 * uo * ss;
      // per element with v = num = O den:  O r = v ir,  dnum = dO / den = ir (Bv w) - bc v
      const float ir = inv * rr, bc = r3 * uo * inv * inv;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        float v[16], fa[16], fb[16];
        tmem_ld16(ta + 16 * j, v);
        unpack8(lds_v4(ogt + sw_off(row, 2 * j)), *reinterpret_cast<float(*)[8]>(fa));
        unpack8(lds_v4(ogt + sw_off(row, 2 * j + 1)), *reinterpret_cast<float(*)[8]>(fa + 8));
        unpack8(lds_v4(dyt + sw_off(row, 2 * j)), *reinterpret_cast<float(*)[8]>(fb));
        unpack8(lds_v4(dyt + sw_off(row, 2 * j + 1)), *reinterpret_cast<float(*)[8]>(fb + 8));
        float wv[16];
        lds_f32n(ws + 64 * j, wv);
        tmem_ld_wait_regs(v);
        float gq[16], gw[16], dn[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const float orr = v[i] * ir;
          gq[i] = fa[i] * orr;
          gw[i] = valid ? fb[i] * orr : 0.f;
          dn[i] = valid ? fmaf(ir, fb[i] * wv[i], -bc * v[i]) : 0.f;
        }
        dnw4[j] += lane_colsum<16>(gw);
        float a[8], c[8];
        if (valid) {
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            a[i] = gq[i];
            c[i] = gq[8 + i];
          }
          __nv_bfloat16 *dst = p.dog + prow0 + (size_t)(li * kKTok + row) * prs + 16 * j;
          *(uint4 *)dst = pack8(a);
          *(uint4 *)(dst + 8) = pack8(c);
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          a[i] = dn[i];
          c[i] = dn[8 + i];
        }
        sts_v4(dnt + sw_off(row, 2 * j), pack8(a));
        sts_v4(dnt + sw_off(row, 2 * j + 1), pack8(c));
      }
      const float dd = valid ? -doo * inv : 0.f;
      fence_proxy_async_smem();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&a1_empty[s]);
        mbar_arrive(&dn_full[s]);
        mbar_arrive(&in_empty[s]);
      }
      // ---- dq~ = (dP + z dden) phi'(q~) and dz, after the dP / dS MMAs
      if (!__all_sync(0xffffffffu, mbar_wait(&a2_full[s], ph, &ab))) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t ta2 = tmem + ((uint32_t)(32 * q4) << 16) + kQA2 + kD * s;
      const uint32_t pt = smem_u32(smem + kQOffP + s * kKTile);
      // this row's P (packed bf16) into registers, so the P stage goes back to
      // the producers before the row is processed
      uint4 prow[8];
#pragma unroll
      for (int c = 0; c < 8; ++c) prow[c] = lds_v4(pt + sw_off(row, c));
      __syncwarp();
      if (lane == 0) mbar_arrive(&p_empty[s]);
      __nv_bfloat16 *dqrow = p.dqt + prow0 + (size_t)(li * kKTok + row) * prs;
#pragma unroll
      for (int part = 0; part < 2; ++part) {
        float v[32];
        tmem_ld16(ta2 + 32 * part, *reinterpret_cast<float(*)[16]>(v));
        tmem_ld16(ta2 + 32 * part + 16, *reinterpret_cast<float(*)[16]>(v + 16));
        tmem_ld_wait();
        if (part == 1) {
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&a2_empty[s]);
        }
        float pz[32];
#pragma unroll
        for (int cq = 0; cq < 4; ++cq) {
          float f[8], z8[8];
          unpack8(prow[4 * part + cq], f);
          lds_f32n(zs + 4 * (32 * part + 8 * cq), z8);
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            pz[8 * cq + e] = f[e] * dd;
            v[8 * cq + e] = (v[8 * cq + e] + z8[e] * dd) * fminf(f[e], 1.f);
          }
          float a[8];
#pragma unroll
          for (int e = 0; e < 8; ++e) a[e] = v[8 * cq + e];
          if (valid) *(uint4 *)(dqrow + 32 * part + 8 * cq) = pack8(a);
        }
        dz2[part] += lane_colsum<32>(pz);
      }
    }
    if (!ok && !ab.raised()) report(512, ab);
  } else if (warp == kQMmaWarp) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t id1 = idesc_bf16_f32(kKTok, 80, 0, 0);
      const uint32_t id2 = idesc_bf16_f32(kKTok, kD, 0, 0);
      const uint32_t id3 = idesc_bf16_f32(kKTok, kD, 1, 1);
      const uint32_t bb = smem_u32(smem + kQOffB);
      bool ok = true;
      auto mma1 = [&](int li) -> bool {
        const int s = li % kKStages;
        tc_fence_after();
        const uint32_t pt = smem_u32(smem + kQOffP + s * kKTile);
#pragma unroll
        for (int k16 = 0; k16 < 4; ++k16) {
          const uint64_t a = sw128_desc(pt + 32 * k16, 16, 1024);
          mma_bf16(tmem + kQA1 + 128 * s, a, sw128_desc(bb + 32 * k16, 16, 1024), id1, k16 != 0);
          mma_bf16(tmem + kQA1 + 128 * s, a, sw128_desc(bb + kQSzT + 32 * k16, 16, 1024), id1, 1);
        }
        mma_commit(&a1_full[s]);
        return true;
      };
      // MMA1 of a tile needs its P tile and a free [num | den] buffer; MMA2 / MMA3
      // need the tile's dnum.  Whichever is ready is issued, so neither waits
      // behind the other.
      auto mma23 = [&](int li) {
        const int s = li % kKStages;
        tc_fence_after();
        const uint32_t dn = smem_u32(smem + kQOffDn + s * kKTile);
        const uint32_t pt = smem_u32(smem + kQOffP + s * kKTile);
#pragma unroll
        for (int k16 = 0; k16 < 4; ++k16) {  // dP = dnum S^T: K = e
          const uint64_t a = sw128_desc(dn + 32 * k16, 16, 1024);
          mma_bf16(tmem + kQA2 + kD * s, a, sw128_desc(bb + 2 * kQSzT + 32 * k16, 16, 1024),
                   id2, k16 != 0);
          mma_bf16(tmem + kQA2 + kD * s, a,
                   sw128_desc(bb + 2 * kQSzT + kKBTile + 32 * k16, 16, 1024), id2, 1);
        }
#pragma unroll
        for (int k16 = 0; k16 < kKTok / 16; ++k16)  // dS += P^T dnum: K = tokens
          mma_bf16(tmem + kQA3, sw128_desc(pt + 2048 * k16, 0, 1024),
                   sw128_desc(dn + 2048 * k16, 16, 1024), id3, (li | k16) != 0);
        mma_commit(&a2_full[s]);
        mma_commit(&dn_empty[s]);
        mma_commit(&p_empty[s]);
      };
      int n1 = 0, n2 = 0;
      uint64_t tw = globaltimer();
      while (ok && n2 < nt) {
        bool moved = false;
        if (n1 < nt) {
          const int s = n1 % kKStages, ph = (n1 / kKStages) & 1;
          if (mbar_try_wait(&p_full[s], ph) && mbar_try_wait(&a1_empty[s], ph ^ 1)) {
            mma1(n1);
            ++n1;
            moved = true;
          }
        }
        if (n2 < n1) {
          const int s = n2 % kKStages, ph = (n2 / kKStages) & 1;
          if (mbar_try_wait(&dn_full[s], ph) && mbar_try_wait(&a2_empty[s], ph ^ 1)) {
            mma23(n2);
            ++n2;
            moved = true;
          }
        }
        if (moved) {
          tw = globaltimer();
        } else if (ab.raised() || globaltimer() - tw > kWaitLimitNs) {
          ok = false;
        }
      }
      if (!ok && !ab.raised()) report(2048, ab);
      mma_commit(a3_full);
      mma_commit(fin);
      if (!mbar_wait(fin, 0, nullptr)) report(4096, ab);
    }
  }
  // every role is done: the input ring is free for the epilogue groups' column
  // sums, then the partial record of this chunk (fixed summation order)
  __syncthreads();
  if (warp >= kQE1Warp0 && warp < kQMmaWarp) {
    const int grp = (warp - kQE1Warp0) >> 2, q4 = warp & 3;
    float *red = (float *)(smem + kQOffIn) + grp * 8 * kD;
    if ((lane & 1) == 0)
#pragma unroll
      for (int j = 0; j < 4; ++j) red[q4 * kD + 16 * j + (lane >> 1)] = dnw4[j];
    red[4 * kD + q4 * kD + lane] = dz2[0];
    red[4 * kD + q4 * kD + 32 + lane] = dz2[1];
  }
  __syncthreads();
  float *rec = p.part + ((size_t)bh * p.nck + chunk) * kQRec;
  const float *red = (const float *)(smem + kQOffIn);
  if (tid < kD) {  // sums over the two groups and four lane quarters in order
    float a = 0.f, w = 0.f;
    for (int g = 0; g < 2; ++g)
      for (int q = 0; q < 4; ++q) {
        w += red[g * 8 * kD + q * kD + tid];
        a += red[g * 8 * kD + 4 * kD + q * kD + tid];
      }
    rec[kD * kD + tid] = a;
    rec[kD * kD + kD + tid] = w;
  }
  if (warp >= kQE2Warp0 && warp < kQMmaWarp && (warp & 3) < 2) {
    // dS rows d = 32 q4 + lane (q4 = 0, 1) from TMEM lanes 0..63
    const int q4 = warp & 3, d = 32 * q4 + lane;
    if (__all_sync(0xffffffffu, nt > 0 && mbar_wait(a3_full, 0, &ab))) {
      tc_fence_after();
      for (int j = 0; j < kD / 16; ++j) {
        float v[16];
        tmem_ld16(tmem + ((uint32_t)(32 * q4) << 16) + kQA3 + 16 * j, v);
        tmem_ld_wait_regs(v);
#pragma unroll
        for (int i = 0; i < 16; ++i) rec[d * kD + 16 * j + i] = v[i];
      }
    } else {
      for (int i = 0; i < kD; ++i) rec[d * kD + i] = 0.f;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == kQMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

using EncodeFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                              const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                              const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                              CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeFn encode() {
  static EncodeFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = (EncodeFn)f;
  });
  return fn;
}

// [B, N, H, 64] bf16 as {D, H, N, B}; box = 64 channels x 1 head x `rows`
// tokens, 128-byte swizzle; rows before 0 or past N read as zeros.
cudaError_t make_rows_map(CUtensorMap *m, const void *base, int B, int N, int H,
                          int rows = kKRawRows) {
  EncodeFn fn = encode();
  if (!fn) return cudaErrorNotSupported;
  const cuuint64_t dims[4] = {(cuuint64_t)kD, (cuuint64_t)H, (cuuint64_t)N, (cuuint64_t)B};
  const cuuint64_t strides[3] = {(cuuint64_t)kD * 2, (cuuint64_t)H * kD * 2,
                                 (cuuint64_t)N * H * kD * 2};
  const cuuint32_t box[4] = {(cuuint32_t)kD, 1, (cuuint32_t)rows, 1};
  const cuuint32_t estr[4] = {1, 1, 1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(base), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

}  // namespace

bool bwd_tc_key_supported(const Problem &p) {
  if (p.dtype != GBLA_BF16 || p.D != kD || p.flags != 0) return false;
  // the key pass indexes its 128-token tiles with an int
  if ((long long)p.B * p.H * ((p.N + kKTok - 1) / kKTok) > 0x7fffffffLL) return false;
  int dev = 0, major = 0, minor = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
  return major == 10 && minor == 3 && encode() != nullptr;
}

cudaError_t bwd_tc_key(const Problem &p, const BwdArgs &a, const float2 *stats,
                       const float *red, const float *dotpart, int ndot, void *dkt,
                       void *dvt, cudaStream_t st) {
  const int BH = p.B * p.H;
  cudaError_t e;
  // rows past seq_lens[b] of dgate are zero; the kernel writes the valid rows
  if (p.seq_lens != nullptr &&
      (e = cudaMemsetAsync(a.dgate, 0, sizeof(__nv_bfloat16) * (size_t)BH * p.N, st)) !=
          cudaSuccess)
    return e;
  CUtensorMap tm_k, tm_v;
  if ((e = make_rows_map(&tm_k, a.k, p.B, p.N, p.H)) != cudaSuccess) return e;
  if ((e = make_rows_map(&tm_v, a.v, p.B, p.N, p.H)) != cudaSuccess) return e;
  KeyParams kp;
  kp.gate = (const __nv_bfloat16 *)a.gate;
  kp.conv_w = a.conv_w;
  kp.stats = stats;
  kp.red = red;
  kp.dotpart = dotpart;
  kp.ndot = ndot;
  kp.seq_lens = p.seq_lens;
  kp.dkt = (__nv_bfloat16 *)dkt;
  kp.dvt = (__nv_bfloat16 *)dvt;
  kp.dgate = (__nv_bfloat16 *)a.dgate;
  kp.B = p.B;
  kp.H = p.H;
  kp.N = p.N;
  kp.tps = (p.N + kKTok - 1) / kKTok;
  if ((e = cudaFuncSetAttribute(tc_bwd_key_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                kKSmem)) != cudaSuccess)
    return e;
  int dev = 0, sms = 1;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const long long tiles = (long long)BH * kp.tps;
  const int grid = (int)(tiles < sms ? tiles : sms);
  if ((e = launch_pdl(tc_bwd_key_kernel, dim3(grid), dim3(kKThreads), (size_t)kKSmem, st, kp,
                      tm_k, tm_v)) != cudaSuccess)
    return e;
  count_launch();
  return cudaGetLastError();
}

// Tiles per query-pass chunk: as few chunks per (b, h) as keep all chunks in
// one wave of one CTA per SM (at least 2 tiles, so the records never outnumber
// the 256-token chunks the scratch layout provides for).
static int bwd_tc_query_tiles(const Problem &p) {
  int dev = 0, sms = 1;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int tps = (p.N + kKTok - 1) / kKTok;
  const int BH = p.B * p.H;
  const int per = sms / BH > 1 ? sms / BH : 1;  // chunks per (b, h)
  const int ct = (tps + per - 1) / per;
  return ct < 2 ? 2 : ct;
}
int bwd_tc_query_chunks(const Problem &p) {
  const int ct = bwd_tc_query_tiles(p), tps = (p.N + kKTok - 1) / kKTok;
  return (tps + ct - 1) / ct;
}

cudaError_t bwd_tc_query(const Problem &p, const BwdArgs &a, const float *state, float *part,
                         void *dqt, cudaStream_t st) {
  const int BH = p.B * p.H;
  cudaError_t e;
  // rows past seq_lens[b] of dout_gate are zero; the kernel writes the valid rows
  if (p.seq_lens != nullptr &&
      (e = cudaMemsetAsync(a.dout_gate, 0, sizeof(__nv_bfloat16) * (size_t)BH * p.N * kD, st)) !=
          cudaSuccess)
    return e;
  CUtensorMap tm_q, tm_og, tm_dy;
  if ((e = make_rows_map(&tm_q, a.q, p.B, p.N, p.H)) != cudaSuccess) return e;
  if ((e = make_rows_map(&tm_og, a.out_gate, p.B, p.N, p.H, kKTok)) != cudaSuccess) return e;
  if ((e = make_rows_map(&tm_dy, a.dy, p.B, p.N, p.H, kKTok)) != cudaSuccess) return e;
  QueryParams qp;
  qp.conv_w = a.conv_w;
  qp.norm_w = a.norm_w;
  qp.state = state;
  qp.seq_lens = p.seq_lens;
  qp.dog = (__nv_bfloat16 *)a.dout_gate;
  qp.dqt = (__nv_bfloat16 *)dqt;
  qp.part = part;
  qp.eps = kRmsEps;
  qp.B = p.B;
  qp.H = p.H;
  qp.N = p.N;
  qp.nck = bwd_tc_query_chunks(p);
  qp.ctiles = bwd_tc_query_tiles(p);
  if ((e = cudaFuncSetAttribute(tc_bwd_query_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                kQSmem)) != cudaSuccess)
    return e;
  if ((e = launch_pdl(tc_bwd_query_kernel, dim3(qp.nck, BH), dim3(kQThreads), (size_t)kQSmem,
                      st, qp, tm_q, tm_og, tm_dy)) != cudaSuccess)
    return e;
  count_launch();
  return cudaGetLastError();
}

unsigned bwd_device_error(bool reset) {
  unsigned v = 0;
  if (cudaMemcpyFromSymbol(&v, g_bwd_error, sizeof(v)) != cudaSuccess) return 0xFFFFFFFFu;
  if (reset) {
    const unsigned z = 0;
    if (cudaMemcpyToSymbol(g_bwd_error, &z, sizeof(z)) != cudaSuccess) return 0xFFFFFFFFu;
  }
  return v;
}

}  // namespace gbla
