// Layer front end on tensor cores (Sec. 2.1 items 1-3), bf16:
//
//   X~ = Conv1D(X)                    depthwise over the d channels, causal, width 4
//   [Q | K | V | R | a] = X~ W^T      one contraction for every head and projection
//
// with the stacked weight matrix W [F, d], F = 4 H D + H: rows s*H*D + h*D + e
// hold output feature (h, e) of stream s = Q, K, V, R (W_R, the output-gate
// input), rows 4 H D + h the gate logits w_g of head h.
//
// tc_project_kernel: persistent, one CTA per SM, 128-token tiles of one
// sequence; each CTA takes an equal run of (tile, 256-column chunk) units.
// Roles:
//  - four converter warps compute X~ for all d channels of a tile in fp32
//    (16-byte loads of the X rows plus 3 rows of history) and store it as
//    bf16 into the K-major A operand: one 128B-swizzled 64-channel block per
//    slot, the whole tile resident (d <= 512);
//  - one warp streams W through a ring of 256-row x 32-channel blocks (TMA,
//    64B swizzle), the same sequence for every tile (W stays in L2);
//  - one thread issues tcgen05.mma (M = 128, N = 256, K = 16, fp32
//    accumulation in TMEM) over the output columns in chunks of 256, two
//    accumulators alternating; the gate logits are a last chunk of N = H
//    rounded up to 16;
//  - four epilogue warps (one per TMEM lane quarter, one token row per
//    thread) round each chunk to bf16 and write it through a per-warp
//    staging buffer as whole 128-byte row segments of q, k, v and out_gate.
// The A slots of a tile are released block by block as the last chunk's MMAs
// finish with them, so the next tile's Conv1D runs under that chunk.
//
// Precision: the Conv1D runs in fp32 (taps in order 0..3, tap 3 on the
// current token) and X~ is rounded once to bf16 for the MMA, the rounding a
// bf16 layer applies between its Conv1D and its projections; products and
// sums are fp32 in the tensor core, and each output is rounded once to bf16.
//
// Every mbarrier wait is bounded (2 s); a wait that runs out sets a bit in
// g_proj_error and the CTA's abort flag, every role leaves its loop, the TMA
// warp waits (bounded) for its copies in flight and the MMA thread for its
// MMAs before TMEM is freed.
#include <mutex>

#include "gbla_internal.cuh"
#include "gbla_sm100.cuh"

namespace gbla {

__device__ unsigned int g_proj_error;

namespace {

using namespace sm100;

constexpr int kPTok = 128;                     // tokens per tile (MMA M)
constexpr int kPChunk = 256;                   // output columns per accumulator (MMA N)
constexpr int kPKB = 64;                       // channels per A block (128-byte rows)
constexpr int kPMaxD = 512;                    // resident A tile: 128 x 512 bf16
constexpr int kPMaxKB = kPMaxD / kPKB;         // 8
constexpr int kPBK = 32;                       // channels per W stage (64-byte rows)
constexpr int kPBStages = 5;
constexpr int kPABlock = kPTok * 128;          // 16384
constexpr int kPBStage = kPChunk * kPBK * 2;   // 16384
constexpr int kPCvtWarps = 4;
constexpr int kPEpiWarps = 4;
constexpr int kPTmaWarp = 0;
constexpr int kPMmaWarp = 1;
constexpr int kPCvtWarp0 = 2;
constexpr int kPEpiWarp0 = kPCvtWarp0 + kPCvtWarps;     // 6
constexpr int kPThreads = (kPEpiWarp0 + kPEpiWarps) * 32;  // 320
constexpr int kPStg = 32 * 128;                // epilogue staging per warp: 32 rows x 64 bf16
constexpr uint32_t kPTmemCols = 2 * kPChunk;   // two accumulators

constexpr int kPOffA = 0;
constexpr int kPOffB = kPOffA + kPMaxKB * kPABlock;         // 131072
constexpr int kPOffStg = kPOffB + kPBStages * kPBStage;     // 212992
constexpr int kPOffBar = kPOffStg + kPEpiWarps * kPStg;     // 229376
// a_full[8], a_empty[8], b_full[5], b_empty[5], acc_full[2], acc_empty[2], fin
constexpr int kPBarCount = 2 * kPMaxKB + 2 * kPBStages + 4 + 1;
constexpr int kPOffMisc = kPOffBar + kPBarCount * 8;       // tmem address, abort flag
constexpr int kPSmemBytes = kPOffMisc + 16 + 1024;         // + alignment slack
static_assert(kPSmemBytes <= 227 * 1024, "projection shared memory");

struct ProjParams {
  const __nv_bfloat16 *x;   // [B, N, d]
  const float *conv_x;      // [d, 4]
  const int32_t *seq_lens;  // [B] or null
  __nv_bfloat16 *q, *k, *v, *og;  // [B, N, H*D]
  __nv_bfloat16 *gate;      // [B, N, H]
  int B, N, d, H, HD;
  int tps;    // tiles per sequence
  int nmain;  // 256-column chunks of q, k, v, out_gate: 4 H D / 256
  int ngate;  // MMA N of the gate chunk: H rounded up to 16
};

// Shared-memory matrix descriptor, 64-byte swizzle (sm_100 layout type 4),
// K-major: 8-row groups `sbo` bytes apart; the leading offset is unused.
__device__ __forceinline__ uint64_t sw64_desc(uint32_t saddr, uint32_t sbo) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr >> 4) & 0x3FFFu);
  d |= (uint64_t)1 << 16;
  d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
  d |= 1ull << 46;
  d |= 4ull << 61;
  return d;
}

__device__ __forceinline__ void report(unsigned code, const AbortFlag &ab) {
  atomicOr(&g_proj_error, code);
  ab.raise();
}

__device__ __forceinline__ int seq_len(const int32_t *seq_lens, int b, int N) {
  if (seq_lens == nullptr) return N;
  const int L = seq_lens[b];
  return L < 0 ? 0 : (L > N ? N : L);
}

// Work is split into units (tile, 256-column chunk of q, k, v, out_gate); the
// gate chunk of a tile goes with the tile's last unit.  CTA c takes the
// contiguous units [c U / G, (c + 1) U / G), U = tiles x chunks, so every CTA
// gets the same number of chunks within one; a tile cut between two CTAs has
// its X~ computed by both.  TileIt walks this CTA's tiles in order, skipping
// tiles that lie wholly in the padding (t0 >= L_b), with the chunk range
// nlo .. nend (nend = the gate chunk when the range reaches the last unit).
struct TileIt {
  int i, b, t0, L, nlo, nend;
};
__device__ __forceinline__ void unit_range(const ProjParams &p, long long &u0, long long &u1) {
  const long long U = (long long)p.B * p.tps * p.nmain;
  u0 = U * blockIdx.x / gridDim.x;
  u1 = U * (blockIdx.x + 1) / gridDim.x;
}
__device__ __forceinline__ bool tile_valid(const ProjParams &p, TileIt &t) {
  long long u0, u1;
  unit_range(p, u0, u1);
  if (u0 >= u1) return false;
  const long long ilast = (u1 - 1) / p.nmain;
  while (t.i <= ilast) {
    t.b = t.i / p.tps;
    t.t0 = (t.i % p.tps) * kPTok;
    t.L = seq_len(p.seq_lens, t.b, p.N);
    if (t.t0 < t.L) {
      t.nlo = t.i == u0 / p.nmain ? (int)(u0 % p.nmain) : 0;
      const int nhi = t.i == ilast ? (int)((u1 - 1) % p.nmain) : p.nmain - 1;
      t.nend = nhi == p.nmain - 1 ? p.nmain : nhi;
      return true;
    }
    ++t.i;
  }
  return false;
}
__device__ __forceinline__ bool tile_first(const ProjParams &p, TileIt &t) {
  long long u0, u1;
  unit_range(p, u0, u1);
  t.i = (int)(u0 / p.nmain);
  return tile_valid(p, t);
}
__device__ __forceinline__ bool tile_next(const ProjParams &p, TileIt &t) {
  ++t.i;
  return tile_valid(p, t);
}

__device__ __forceinline__ void unpack8(uint4 r, float (&f)[8]) {
  const float2 a = bf2_to_f2(r.x), b = bf2_to_f2(r.y), c = bf2_to_f2(r.z), d = bf2_to_f2(r.w);
  f[0] = a.x; f[1] = a.y; f[2] = b.x; f[3] = b.y;
  f[4] = c.x; f[5] = c.y; f[6] = d.x; f[7] = d.y;
}

// One converter unit: 8 channels (c0 .. c0 + 7) x 8 tile rows (8 rg .. 8 rg + 7)
// of one 64-channel block; raw[j] holds X row t0 + 8 rg - 3 + j.
struct CvtUnit {
  TileIt t;
  int kb, tseq;  // 64-channel block; tile sequence number within this CTA
  bool valid;
};

__global__ void __launch_bounds__(kPThreads, 1)
    tc_project_kernel(const ProjParams p, const __grid_constant__ CUtensorMap tm_w) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nkb = p.d / kPKB;

  uint64_t *bars = (uint64_t *)(smem + kPOffBar);
  uint64_t *a_full = bars, *a_empty = bars + kPMaxKB;
  uint64_t *b_full = bars + 2 * kPMaxKB, *b_empty = b_full + kPBStages;
  uint64_t *acc_full = b_empty + kPBStages, *acc_empty = acc_full + 2;
  uint64_t *fin = acc_empty + 2;
  uint32_t *tmem_slot = (uint32_t *)(smem + kPOffMisc);
  const AbortFlag ab{smem_u32(smem + kPOffMisc + 4)};

  TileIt t0;
  if (!tile_first(p, t0)) return;  // no work for this CTA (uniform over the block)

  if (tid == 0) {
    for (int i = 0; i < kPMaxKB; ++i) {
      mbar_init(&a_full[i], kPCvtWarps);
      mbar_init(&a_empty[i], 1);
    }
    for (int i = 0; i < kPBStages; ++i) {
      mbar_init(&b_full[i], 1);
      mbar_init(&b_empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], kPEpiWarps);
    }
    mbar_init(fin, 1);
    *(volatile int *)(smem + kPOffMisc + 4) = 0;
    fence_mbar_init();
  }
  if (warp == kPTmaWarp && lane == 0) tma_prefetch_desc(&tm_w);
  if (warp == kPMmaWarp) tmem_alloc(tmem_slot, kPTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == kPTmaWarp) {
    // ------------------------------------------------------------ TMA: W blocks
    if (lane == 0) {
      const uint64_t pol = l2_policy_evict_last();  // every CTA reads W once per tile
      int bs = 0;
      bool ok = true;
      TileIt t = t0;
      do {
        for (int n = t.nlo; n <= t.nend && ok; ++n)
          for (int kb = 0; kb < nkb && ok; ++kb)
            for (int half = 0; half < 2; ++half) {
              const int s = bs % kPBStages;
              if (!mbar_wait(&b_empty[s], ((bs / kPBStages) & 1) ^ 1, &ab)) {
                if (!ab.raised()) report(1, ab);
                ok = false;
                break;
              }
              mbar_arrive_expect_tx(&b_full[s], kPBStage);
              tma_load_4d_hint(smem + kPOffB + s * kPBStage, &tm_w, &b_full[s],
                               kb * kPKB + half * kPBK, n * kPChunk, 0, 0, pol);
              ++bs;
            }
      } while (ok && tile_next(p, t));
      // the copies still in flight land before the CTA can end
      for (int j = bs > kPBStages ? bs - kPBStages : 0; j < bs; ++j)
        if (!mbar_wait(&b_full[j % kPBStages], (j / kPBStages) & 1, nullptr)) report(2, ab);
    }
  } else if (warp == kPMmaWarp) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t id_main = idesc_bf16_f32(kPTok, kPChunk, 0, 0);
      const uint32_t id_gate = idesc_bf16_f32(kPTok, p.ngate, 0, 0);
      // The loop is kept short (this warp shares its sub-partition with busy
      // converter and epilogue warps): descriptors of block 0 / stage 0 are
      // advanced by byte offsets (the address field is the byte address >> 4
      // and shared addresses stay below 256 KB, so adding never carries into
      // the next field), and ring positions are stepped rather than divided.
      const uint64_t ad0 = sw128_desc(smem_u32(smem + kPOffA), 16, 1024);
      const uint64_t bd0 = sw64_desc(smem_u32(smem + kPOffB), 512);
      int bstage = 0, bphase = 0, cs = 0, tseq = 0;
      bool ok = true;
      TileIt t = t0;
      do {
        for (int n = t.nlo; n <= t.nend && ok; ++n) {
          const int buf = cs & 1;
          if (!mbar_wait(&acc_empty[buf], ((cs >> 1) & 1) ^ 1, &ab)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t dacc = tmem + buf * kPChunk;
          const uint32_t idesc = n < p.nmain ? id_main : id_gate;
          const bool first = n == t.nlo, last = n == t.nend;
          for (int kb = 0; kb < nkb && ok; ++kb) {
            if (first && !mbar_wait(&a_full[kb], tseq & 1, &ab)) {
              ok = false;
              break;
            }
            const uint64_t adk = ad0 + (uint64_t)((kb * kPABlock) >> 4);
#pragma unroll
            for (int half = 0; half < 2; ++half) {
              if (!mbar_wait(&b_full[bstage], bphase, &ab)) {
                ok = false;
                break;
              }
              tc_fence_after();
              const uint64_t bds = bd0 + (uint64_t)((bstage * kPBStage) >> 4);
              mma_bf16(dacc, adk + (uint64_t)((half * 64) >> 4), bds, idesc, (kb | half) != 0);
              mma_bf16(dacc, adk + (uint64_t)((half * 64 + 32) >> 4), bds + 2, idesc, 1);
              mma_commit(&b_empty[bstage]);
              if (++bstage == kPBStages) {
                bstage = 0;
                bphase ^= 1;
              }
            }
            if (ok && last) mma_commit(&a_empty[kb]);
          }
          if (ok) mma_commit(&acc_full[buf]);
          ++cs;
        }
        ++tseq;
      } while (ok && tile_next(p, t));
      if (!ok && !ab.raised()) report(4, ab);
      mma_commit(fin);  // every MMA issued above has completed once this arrives
      if (!mbar_wait(fin, 0, nullptr)) report(8, ab);
    }
  } else if (warp < kPEpiWarp0) {
    // ------------------------------------------------------------ converters: Conv1D of X
    const int ct = tid - kPCvtWarp0 * 32;  // 0..127
    const int cg = ct & 7, rg = ct >> 3;   // 16-byte channel chunk, 8-row group
    const size_t d = (size_t)p.d;
    auto load = [&](const CvtUnit &u, uint4 (&raw)[11]) {
      const __nv_bfloat16 *xp = p.x + (size_t)u.t.b * p.N * d + u.kb * kPKB + cg * 8;
      const int ts = u.t.t0 + rg * 8 - 3, tmax = u.t.L - 1;
#pragma unroll
      for (int j = 0; j < 11; ++j) {
        const int t = ts + j;
        raw[j] = t < 0 ? make_uint4(0u, 0u, 0u, 0u) : ldg_nc_v4(xp + (size_t)min(t, tmax) * d);
      }
    };
    auto advance = [&](CvtUnit u) {
      if (++u.kb == nkb) {
        u.kb = 0;
        ++u.tseq;
        u.valid = tile_next(p, u.t);
      }
      return u;
    };
    auto convert = [&](const CvtUnit &u, const uint4 (&raw)[11]) -> bool {
      const int c0 = u.kb * kPKB + cg * 8;
      if (u.kb == 0 && ct == 0) {
        // warm L2 with the next tile's X rows (read by this role one tile later)
        TileIt nx = u.t;
        if (tile_next(p, nx)) {
          const char *src = (const char *)(p.x + ((size_t)nx.b * p.N + (nx.t0 > 3 ? nx.t0 - 3 : 0)) * d);
          const int rows = min(nx.L - nx.t0, kPTok) + (nx.t0 > 3 ? 3 : nx.t0);
          const uint32_t bytes = (uint32_t)(rows * d * 2);
          for (uint32_t o = 0; o < bytes; o += 16384)
            prefetch_l2(src + o, min(16384u, bytes - o));
        }
      }
      float4 tap[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) tap[i] = __ldg((const float4 *)(p.conv_x + (size_t)(c0 + i) * 4));
      if (!mbar_wait(&a_empty[u.kb], (u.tseq & 1) ^ 1, &ab)) return false;
      const uint32_t ab0 = smem_u32(smem + kPOffA + u.kb * kPABlock) + rg * 1024;
      float h0[8], h1[8], h2[8];
      unpack8(raw[0], h0);
      unpack8(raw[1], h1);
      unpack8(raw[2], h2);
#pragma unroll
      for (int r = 0; r < 8; ++r) {
        float cur[8], y[8];
        unpack8(raw[r + 3], cur);
#pragma unroll
        for (int i = 0; i < 8; ++i)
          y[i] = fmaf(tap[i].w, cur[i], fmaf(tap[i].z, h2[i], fmaf(tap[i].y, h1[i], tap[i].x * h0[i])));
        sts_v4(ab0 + r * 128 + ((cg ^ r) << 4),
               make_uint4(f2_to_bf2(y[0], y[1]), f2_to_bf2(y[2], y[3]), f2_to_bf2(y[4], y[5]),
                          f2_to_bf2(y[6], y[7])));
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          h0[i] = h1[i];
          h1[i] = h2[i];
          h2[i] = cur[i];
        }
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&a_full[u.kb]);
      return true;
    };
    CvtUnit cur{t0, 0, 0, true};
    uint4 ra[11], rb[11];
    load(cur, ra);
    bool ok = true;
    while (cur.valid && ok) {
      CvtUnit nx = advance(cur);
      if (nx.valid) load(nx, rb);
      ok = convert(cur, ra);
      cur = nx;
      if (!cur.valid || !ok) break;
      nx = advance(cur);
      if (nx.valid) load(nx, ra);
      ok = convert(cur, rb);
      cur = nx;
    }
    if (!ok && !ab.raised()) report(16, ab);
  } else {
    // ------------------------------------------------------------ epilogue
    const int ew = warp - kPEpiWarp0;
    const int q4 = warp & 3;  // TMEM lane quarter this warp may access
    const int row = 32 * q4 + lane;
    const uint32_t stg = smem_u32(smem + kPOffStg + ew * kPStg);
    const int HD = p.HD;
    int cs = 0;
    bool ok = true;
    TileIt t = t0;
    do {
      const size_t tok0 = (size_t)t.b * p.N + t.t0;  // token index of tile row 0
      for (int n = t.nlo; n <= t.nend; ++n, ++cs) {
        const int buf = cs & 1;
        if (!mbar_wait(&acc_full[buf], (cs >> 1) & 1, &ab)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t tacc = tmem + ((uint32_t)(32 * q4) << 16) + buf * kPChunk;
        if (n < p.nmain) {
#pragma unroll 1
          for (int g = 0; g < kPChunk / 64; ++g) {
            float v[4][16];
#pragma unroll
            for (int j = 0; j < 4; ++j) tmem_ld16(tacc + g * 64 + 16 * j, v[j]);
            tmem_ld_wait_regs(v[0]);
            tmem_ld_wait_regs(v[1]);
            tmem_ld_wait_regs(v[2]);
            tmem_ld_wait_regs(v[3]);
            if (g == kPChunk / 64 - 1) {  // accumulator drained: hand it back
              tc_fence_before();
              __syncwarp();
              if (lane == 0) mbar_arrive(&acc_empty[buf]);
            }
            // this row's 64 values -> 8 swizzled 16-byte pieces of the staging row
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              const float *f = &v[j >> 1][(j & 1) * 8];
              sts_v4(stg + lane * 128 + ((j ^ (lane & 7)) << 4),
                     make_uint4(f2_to_bf2(f[0], f[1]), f2_to_bf2(f[2], f[3]),
                                f2_to_bf2(f[4], f[5]), f2_to_bf2(f[6], f[7])));
            }
            __syncwarp();
            const int gcol = n * kPChunk + g * 64;
            const int s = gcol / HD, col = gcol % HD;
            __nv_bfloat16 *dst = s == 0 ? p.q : s == 1 ? p.k : s == 2 ? p.v : p.og;
            // 4 rows x 128 bytes per warp store
#pragma unroll
            for (int it = 0; it < 8; ++it) {
              const int rr = it * 4 + (lane >> 3), ch = lane & 7;
              const uint4 val = lds_v4(stg + rr * 128 + ((ch ^ (rr & 7)) << 4));
              const int trow = 32 * q4 + rr;
              if (t.t0 + trow < t.L)
                *(uint4 *)(dst + (tok0 + trow) * HD + col + ch * 8) = val;
            }
            __syncwarp();
          }
        } else {
          // gate logits: H columns, stored per row
          const bool valid = t.t0 + row < t.L;
          __nv_bfloat16 *gp = p.gate + (tok0 + row) * p.H;
          for (int h0 = 0; h0 < p.ngate; h0 += 16) {
            float v[16];
            tmem_ld16(tacc + h0, v);
            tmem_ld_wait_regs(v);
            if (valid)
#pragma unroll
              for (int j = 0; j < 16; ++j)
                if (h0 + j < p.H) gp[h0 + j] = __float2bfloat16_rn(v[j]);
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&acc_empty[buf]);
        }
      }
    } while (ok && tile_next(p, t));
    if (!ok && !ab.raised()) report(32, ab);
  }
  __syncthreads();
  if (warp == kPMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem, kPTmemCols);
  }
}

}  // namespace

// W [F, d] bf16 as a 4-D map {d, F, 1, 1}; box = 32 channels x 256 rows,
// 64-byte swizzle (the B-operand layout of the kernel's MMAs).  Rows past F
// read as zeros.
static cudaError_t make_w_map(CUtensorMap *m, const void *w, int F, int d) {
  using EncodeFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
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
  if (!fn) return cudaErrorNotSupported;
  const cuuint64_t dims[4] = {(cuuint64_t)d, (cuuint64_t)F, 1, 1};
  const cuuint64_t strides[3] = {(cuuint64_t)d * 2, (cuuint64_t)F * d * 2,
                                 (cuuint64_t)F * d * 2};
  const cuuint32_t box[4] = {(cuuint32_t)kPBK, (cuuint32_t)kPChunk, 1, 1};
  const cuuint32_t estr[4] = {1, 1, 1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(w), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

bool project_supports(const ProjProblem &pp) {
  if (pp.d < kPKB || pp.d > kPMaxD || pp.d % kPKB != 0) return false;
  if ((pp.H * pp.D) % 64 != 0 || pp.H > kPChunk) return false;
  int dev = 0, major = 0, minor = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
  return major == 10 && minor == 3;
}

cudaError_t tc_project(const ProjProblem &pp, const void *x, const float *conv_x,
                       const void *w, void *q, void *k, void *v, void *og, void *gate,
                       cudaStream_t st) {
  ProjParams p;
  p.x = (const __nv_bfloat16 *)x;
  p.conv_x = conv_x;
  p.seq_lens = pp.seq_lens;
  p.q = (__nv_bfloat16 *)q;
  p.k = (__nv_bfloat16 *)k;
  p.v = (__nv_bfloat16 *)v;
  p.og = (__nv_bfloat16 *)og;
  p.gate = (__nv_bfloat16 *)gate;
  p.B = pp.B;
  p.N = pp.N;
  p.d = pp.d;
  p.H = pp.H;
  p.HD = pp.H * pp.D;
  p.tps = (pp.N + kPTok - 1) / kPTok;
  p.nmain = 4 * p.HD / kPChunk;
  p.ngate = (pp.H + 15) / 16 * 16;
  const int F = 4 * p.HD + pp.H;
  CUtensorMap tm_w;
  cudaError_t e = make_w_map(&tm_w, w, F, pp.d);
  if (e != cudaSuccess) return e;
  if ((e = cudaFuncSetAttribute(tc_project_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                kPSmemBytes)) != cudaSuccess)
    return e;
  int dev = 0, sms = 1;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const long long units = (long long)pp.B * p.tps * p.nmain;
  const int grid = (int)(units < sms ? units : sms);
  tc_project_kernel<<<grid, kPThreads, kPSmemBytes, st>>>(p, tm_w);
  count_launch();
  return cudaGetLastError();
}

unsigned project_device_error(bool reset) {
  unsigned v = 0;
  if (cudaMemcpyFromSymbol(&v, g_proj_error, sizeof(v)) != cudaSuccess) return 0xFFFFFFFFu;
  if (reset) {
    const unsigned z = 0;
    if (cudaMemcpyToSymbol(g_proj_error, &z, sizeof(z)) != cudaSuccess) return 0xFFFFFFFFu;
  }
  return v;
}

}  // namespace gbla
