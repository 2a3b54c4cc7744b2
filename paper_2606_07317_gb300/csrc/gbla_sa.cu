// Bidirectional softmax attention (Sec. 2, "Bidirectional softmax attention"):
// the SA layer of the paper's hybrid [SA, LA, LA] encoder (Sec. 3), against
// which the GBLA layer's latency is compared (Sec. 4, Table 5).  For every
// valid query i < L of a (batch, head),
//   o_i = sum_j exp(q_i . k_j / sqrt(d_h)) v_j / sum_j exp(q_i . k_j / sqrt(d_h))
// over the valid keys j < L.  bf16 inputs and output, d_h = 64, fp32
// accumulation, on tcgen05 tensor cores.
//
// One CTA per 128-query tile of one (batch, head); the keys go by in blocks of
// 128.  Six warps:
//   warps 0-3  softmax: one query row per thread (its TMEM lane).  They read
//              the block's scores S = Q K^T from TMEM, keep a running row
//              maximum m and sum l, write P = 2^((s - m) log2(e) / sqrt(d_h))
//              as bf16 into a 128B-swizzled K-major tile, and at the end divide
//              O by l and store it.  The maximum is lazy: O and l are rescaled
//              (in TMEM) only when the row maximum grows by more than 2^8 in
//              probability, otherwise the old maximum stays and P <= 2^8.
//   warp 4     MMA issuer: S_j = Q K_j^T (M128 N128 K64) into one of two TMEM
//              score buffers, then O += P_{j-1} V_{j-1} (M128 N64 K128, V as
//              an MN-major operand straight from its TMA tile), so the scores
//              of block j are computed while the softmax works on block j-1.
//   warp 5     TMA: Q once, then K and V blocks through a 3-deep ring.
// Keys past the sequence end get score -inf and their V rows are zeroed in
// shared memory (the padding may hold NaN, which a zero probability does not
// cancel); queries past the end are computed but not stored.
//
// Every mbarrier wait is bounded (2 s, as in the GBLA kernels); a wait that
// runs out records a bit in g_sa_error and raises the CTA's abort flag.
#include <math.h>

#include <mutex>

#include "gbla_internal.cuh"
#include "gbla_sm100.cuh"

namespace gbla {

__device__ unsigned int g_sa_error;

namespace {

using namespace sm100;

constexpr int kQ = 128;      // queries per CTA (MMA M)
constexpr int kKey = 128;    // keys per block
constexpr int kDh = 64;      // head dimension
constexpr int kSmWarps = 4;  // softmax warps
constexpr int kMmaWarp = 4, kTmaWarp = 5;
constexpr int kThreads = 6 * 32;
constexpr int kKV = 3;       // K/V ring depth
constexpr int kTile = kQ * kDh * 2;          // 16 KB: a 128 x 64 bf16 tile
constexpr int kPBuf = kQ * kKey * 2;         // 32 KB: P as two 64-key K blocks
constexpr int kOffQ = 0;
constexpr int kOffK = kOffQ + kTile;
constexpr int kOffV = kOffK + kKV * kTile;
constexpr int kOffP = kOffV + kKV * kTile;
constexpr int kOffBar = kOffP + 2 * kPBuf;
// q_full, kv_full[3], kv_empty[3], s_full[2], s_empty[2], p_full[2], p_empty[2], o_ready
constexpr int kBars = 1 + 2 * kKV + 8 + 1;
constexpr int kOffMisc = kOffBar + kBars * 8;
constexpr int kSmem = kOffMisc + 16 + 1024;
static_assert(kSmem <= 227 * 1024, "attention shared memory");
constexpr uint32_t kTmemCols = 512;  // S0 [0,128), S1 [128,256), O [256,320)
constexpr uint32_t kOCol = 256;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLazy = 8.f;  // rescale only when the maximum grows by more than 2^8
constexpr int kPolyEvery = 4;  // every fourth pair of exponentials on the FMA pipe

// 2^x for two values on the FMA and integer pipes (no special-function op):
// x = n + f with n = round(x) (the 1.5 * 2^23 addition leaves n in the low
// mantissa bits) and f in [-1/2, 1/2]; 2^f by a cubic fitted here to 2^f on
// [-1/2, 1/2] (least squares on the relative error, reweighted towards its
// maximum; maximum relative error 7.6e-5, far below the 2^-9 of the bf16
// rounding every probability gets); n added to the exponent field.  x is
// clamped at -125 (2^-125 stands in for 0: past-the-end keys meet zeroed V
// rows, and the sum of P is at least 1).
__device__ __forceinline__ float2 exp2_poly2(float2 x) {
  constexpr float kRound = 12582912.f;  // 1.5 * 2^23
  x = make_float2(fmaxf(x.x, -125.f), fmaxf(x.y, -125.f));
  const float2 t = __fadd2_rn(x, make_float2(kRound, kRound));
  const float2 r = __fadd2_rn(t, make_float2(-kRound, -kRound));  // n as a float
  const float2 f = __ffma2_rn(r, make_float2(-1.f, -1.f), x);        // x - n
  float2 q = __ffma2_rn(make_float2(0.05517030f, 0.05517030f), f,
                        make_float2(0.24260803f, 0.24260803f));
  q = __ffma2_rn(q, f, make_float2(0.69326091f, 0.69326091f));
  q = __ffma2_rn(q, f, make_float2(0.99992830f, 0.99992830f));
  // bits(t) << 23 = n << 23 (mod 2^32): the rounding constant's own bits shift out
  return make_float2(__int_as_float(__float_as_int(q.x) + (__float_as_int(t.x) << 23)),
                     __int_as_float(__float_as_int(q.y) + (__float_as_int(t.y) << 23)));
}

struct SaParams {
  const int32_t *seq_lens;
  __nv_bfloat16 *o;
  int B, H, N;
};

__device__ __forceinline__ void sa_error(unsigned code, const AbortFlag &ab) {
  atomicOr(&g_sa_error, code);
  ab.raise();
}

__device__ __forceinline__ void tmem_st16(uint32_t taddr, const float (&v)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(taddr),
      "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])),
      "r"(__float_as_uint(v[3])), "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])),
      "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])), "r"(__float_as_uint(v[8])),
      "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
      "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
      "r"(__float_as_uint(v[15]))
      : "memory");
}
__device__ __forceinline__ void tmem_st_wait() {
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

__global__ void __launch_bounds__(kThreads, 1)
    sa_kernel(const SaParams p, const __grid_constant__ CUtensorMap tm_q,
              const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint64_t *bars = (uint64_t *)(smem + kOffBar);
  uint64_t *q_full = bars, *kv_full = bars + 1, *kv_empty = kv_full + kKV;
  uint64_t *s_full = kv_empty + kKV, *s_empty = s_full + 2, *p_full = s_empty + 2,
           *p_empty = p_full + 2, *o_ready = p_empty + 2;
  uint32_t *tmem_slot = (uint32_t *)(smem + kOffMisc);
  const AbortFlag ab{smem_u32(smem + kOffMisc + 4)};

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int qt = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int L = p.seq_lens == nullptr ? p.N : min(max(p.seq_lens[b], 0), p.N);
  const int q0 = qt * kQ;
  if (q0 >= L) return;  // no valid query in this tile
  const int nb = (L + kKey - 1) / kKey;

  if (tid == 0) {
    *(volatile int *)(smem + kOffMisc + 4) = 0;
    mbar_init(q_full, 1);
    for (int i = 0; i < kKV; ++i) {
      mbar_init(&kv_full[i], 1);
      mbar_init(&kv_empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s_full[i], 1);
      mbar_init(&s_empty[i], kSmWarps);
      mbar_init(&p_full[i], kSmWarps);
      mbar_init(&p_empty[i], 1);
    }
    mbar_init(o_ready, 1);
    fence_mbar_init();
  }
  if (warp == kTmaWarp && lane == 0) {
    tma_prefetch_desc(&tm_q);
    tma_prefetch_desc(&tm_k);
    tma_prefetch_desc(&tm_v);
  }
  if (warp == kMmaWarp) tmem_alloc(tmem_slot, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == kTmaWarp) {
    // -------------------------------------------------------------- TMA
    if (lane == 0) {
      const uint64_t pol = l2_policy_evict_last();  // K and V are read by every query tile
      mbar_arrive_expect_tx(q_full, kTile);
      tma_load_4d(smem + kOffQ, &tm_q, q_full, 0, h, q0, b);
      for (int j = 0; j < nb; ++j) {
        const int st = j % kKV;
        if (!mbar_wait(&kv_empty[st], ((j / kKV) & 1) ^ 1, &ab)) {
          if (!ab.raised()) sa_error(1, ab);
          break;
        }
        mbar_arrive_expect_tx(&kv_full[st], 2 * kTile);
        tma_load_4d_hint(smem + kOffK + st * kTile, &tm_k, &kv_full[st], 0, h, j * kKey, b, pol);
        tma_load_4d_hint(smem + kOffV + st * kTile, &tm_v, &kv_full[st], 0, h, j * kKey, b, pol);
      }
    }
  } else if (warp == kMmaWarp) {
    // -------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc_qk = idesc_bf16_f32(kQ, kKey, 0, 0);  // Q, K both K-major
      constexpr uint32_t idesc_pv = idesc_bf16_f32(kQ, kDh, 0, 1);   // P K-major, V MN-major
      const uint32_t qs = smem_u32(smem + kOffQ), ks = smem_u32(smem + kOffK),
                     vs = smem_u32(smem + kOffV), ps = smem_u32(smem + kOffP);
      bool ok = mbar_wait(q_full, 0, &ab);
      for (int j = 0; j <= nb && ok; ++j) {
        if (j < nb) {
          const int st = j % kKV;
          ok = mbar_wait(&kv_full[st], (j / kKV) & 1, &ab);
          if (ok && j >= 2) ok = mbar_wait(&s_empty[j & 1], ((j - 2) >> 1) & 1, &ab);
          if (!ok) break;
          tc_fence_after();
#pragma unroll
          for (int k16 = 0; k16 < kDh / 16; ++k16)
            mma_bf16(tmem + (uint32_t)(kKey * (j & 1)), sw128_desc(qs + k16 * 32, 16, 1024),
                     sw128_desc(ks + st * kTile + k16 * 32, 16, 1024), idesc_qk, k16 != 0);
          mma_commit(&s_full[j & 1]);
        }
        if (j >= 1) {
          const int jp = j - 1, st = jp % kKV;
          if (!(ok = mbar_wait(&p_full[jp & 1], (jp >> 1) & 1, &ab))) break;
          tc_fence_after();
          const uint32_t pb = ps + (jp & 1) * kPBuf;
#pragma unroll
          for (int k16 = 0; k16 < kKey / 16; ++k16)
            mma_bf16(tmem + kOCol, sw128_desc(pb + (k16 >> 2) * (kQ * 128) + (k16 & 3) * 32, 16, 1024),
                     sw128_desc(vs + st * kTile + k16 * 16 * 128, 8192, 1024), idesc_pv,
                     (jp | k16) != 0);
          mma_commit(&p_empty[jp & 1]);
          mma_commit(&kv_empty[st]);
        }
      }
      if (!ok && !ab.raised()) sa_error(2, ab);
      mma_commit(o_ready);  // every MMA issued above has completed once this arrives
    }
  } else {
    // -------------------------------------------------------------- softmax
    const int row = tid;  // query q0 + row, TMEM lane row
    const uint32_t tl = tmem + ((uint32_t)(32 * warp) << 16);
    const float c = kLog2e / sqrtf((float)kDh);  // scores to log2 units
    float m_run = -INFINITY, l_run = 0.f;        // in log2 units (m) / probability (l)
    const uint32_t ps = smem_u32(smem + kOffP);
    for (int j = 0; j < nb; ++j) {
      const int sb = j & 1;
      if (!mbar_wait(&s_full[sb], (j >> 1) & 1, &ab) && !ab.raised()) sa_error(4, ab);
      tc_fence_after();
      float sv[kKey];
#pragma unroll
      for (int i = 0; i < kKey / 16; ++i) {
        float t16[16];
        tmem_ld16(tl + (uint32_t)(kKey * sb + 16 * i), t16);
#pragma unroll
        for (int e = 0; e < 16; ++e) sv[16 * i + e] = t16[e];
      }
      tmem_ld_wait_regs(sv);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&s_empty[sb]);  // the score buffer may be overwritten
      const int kv_valid = L - j * kKey;           // keys of this block before the end
      if (kv_valid < kKey) {                       // the last block: keys past the end
#pragma unroll
        for (int i = 0; i < kKey; ++i) sv[i] = i < kv_valid ? sv[i] : -INFINITY;
      }
      float mb = -INFINITY;  // the row maximum of the raw scores, then in log2 units (c > 0)
#pragma unroll
      for (int i = 0; i < kKey; i += 2) mb = fmaxf(mb, fmaxf(sv[i], sv[i + 1]));
      mb *= c;
      // The row maximum grew: rescale O and l (lazily).  TMEM loads and stores
      // are warp-wide, so the whole warp takes the O pass when any lane needs
      // it, with alpha = 1 on the other lanes.
      const bool grow = mb > m_run + kLazy;
      if (j > 0 && __any_sync(0xffffffffu, grow)) {
        // O is stable once the previous block's P V has completed
        if (!mbar_wait(&p_empty[(j - 1) & 1], ((j - 1) >> 1) & 1, &ab) && !ab.raised())
          sa_error(8, ab);
        tc_fence_after();
        const float alpha = grow ? ex2_approx(m_run - mb) : 1.f;
#pragma unroll
        for (int i = 0; i < kDh / 16; ++i) {
          float o16[16];
          tmem_ld16(tl + kOCol + 16 * i, o16);
          tmem_ld_wait_regs(o16);
#pragma unroll
          for (int e = 0; e < 16; ++e) o16[e] *= alpha;
          tmem_st16(tl + kOCol + 16 * i, o16);
        }
        tmem_st_wait();
        l_run *= alpha;
      }
      if (grow) m_run = mb;
      // P = 2^(s c - m) (at most 2^8 with the lazy maximum), every kPolyEvery-th
      // pair by the polynomial, the others by ex2; the sum in fp32
      float2 ls2 = make_float2(0.f, 0.f);
#pragma unroll
      for (int i = 0; i < kKey; i += 2) {
        const float2 x = __ffma2_rn(make_float2(sv[i], sv[i + 1]), make_float2(c, c),
                                    make_float2(-m_run, -m_run));
        const float2 e = (i / 2) % kPolyEvery == kPolyEvery - 1
                             ? exp2_poly2(x)
                             : make_float2(ex2_approx(x.x), ex2_approx(x.y));
        sv[i] = e.x;
        sv[i + 1] = e.y;
        ls2 = __fadd2_rn(ls2, e);
      }
      l_run += ls2.x + ls2.y;
      if (j >= 2 && !mbar_wait(&p_empty[sb], ((j - 2) >> 1) & 1, &ab) && !ab.raised())
        sa_error(16, ab);  // the P buffer is free once the P V of block j - 2 is done
      // row `row` of P: two 64-key K blocks, 16-byte chunks swizzled by the row
      const uint32_t pr = ps + sb * kPBuf + (row >> 3) * 1024 + (row & 7) * 128;
#pragma unroll
      for (int ch = 0; ch < kKey / 8; ++ch) {
        const int kb = ch >> 3, cc = ch & 7;
        sts_v4(pr + kb * (kQ * 128) + ((cc ^ (row & 7)) << 4),
               make_uint4(f2_to_bf2(sv[8 * ch], sv[8 * ch + 1]), f2_to_bf2(sv[8 * ch + 2], sv[8 * ch + 3]),
                          f2_to_bf2(sv[8 * ch + 4], sv[8 * ch + 5]),
                          f2_to_bf2(sv[8 * ch + 6], sv[8 * ch + 7])));
      }
      if (j == nb - 1 && kv_valid < kKey) {
        // V rows of keys past the end meet P = 0, but may hold NaN: zero them
        const int st = j % kKV;
        if (!mbar_wait(&kv_full[st], (j / kKV) & 1, &ab) && !ab.raised()) sa_error(32, ab);
        const uint32_t vb = smem_u32(smem + kOffV + st * kTile);
        for (int e = tid; e < (kKey - kv_valid) * 8; e += kSmWarps * 32)
          sts_v4(vb + (kv_valid + e / 8) * 128 + (e % 8) * 16, make_uint4(0, 0, 0, 0));
      }
      fence_proxy_async_smem();  // P (and zeroed V rows) visible to the tensor cores
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&p_full[sb]);
    }
    // ---- epilogue: O / l, one bf16 row per thread (valid queries only)
    if (!mbar_wait(o_ready, 0, &ab) && !ab.raised()) sa_error(64, ab);
    tc_fence_after();
    float ov[kDh];
#pragma unroll
    for (int i = 0; i < kDh / 16; ++i) {
      float o16[16];
      tmem_ld16(tl + kOCol + 16 * i, o16);
#pragma unroll
      for (int e = 0; e < 16; ++e) ov[16 * i + e] = o16[e];
    }
    tmem_ld_wait_regs(ov);
    const float inv = l_run > 0.f ? 1.f / l_run : 0.f;
    if (q0 + row < L) {
      uint4 *dst = (uint4 *)(p.o + (((size_t)b * p.N + q0 + row) * p.H + h) * kDh);
#pragma unroll
      for (int ch = 0; ch < kDh / 8; ++ch)
        dst[ch] = make_uint4(f2_to_bf2(ov[8 * ch] * inv, ov[8 * ch + 1] * inv),
                             f2_to_bf2(ov[8 * ch + 2] * inv, ov[8 * ch + 3] * inv),
                             f2_to_bf2(ov[8 * ch + 4] * inv, ov[8 * ch + 5] * inv),
                             f2_to_bf2(ov[8 * ch + 6] * inv, ov[8 * ch + 7] * inv));
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                   const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                   const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn sa_encode_fn() {
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

// 4-D map over a [B, N, H, 64] bf16 tensor: box = 64 channels x 1 head x 128
// tokens, 128-byte swizzle (K-major Q and K tiles, MN-major V tile).
cudaError_t sa_map(CUtensorMap *m, const void *base, int B, int N, int H) {
  EncodeTiledFn fn = sa_encode_fn();
  if (!fn) return cudaErrorNotSupported;
  const cuuint64_t dims[4] = {(cuuint64_t)kDh, (cuuint64_t)H, (cuuint64_t)N, (cuuint64_t)B};
  const cuuint64_t strides[3] = {(cuuint64_t)kDh * 2, (cuuint64_t)H * kDh * 2,
                                 (cuuint64_t)N * H * kDh * 2};
  const cuuint32_t box[4] = {kDh, 1, kQ, 1};
  const cuuint32_t estr[4] = {1, 1, 1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(base), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

}  // namespace

bool sa_supports(int D, gbla_dtype dtype) {
  if (dtype != GBLA_BF16 || D != kDh) return false;
  int dev = 0, major = 0, minor = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
  return major == 10 && minor == 3 && sa_encode_fn() != nullptr;
}

cudaError_t sa_forward(const void *q, const void *k, const void *v, const int32_t *seq_lens,
                       void *o, int B, int H, int N, cudaStream_t st) {
  CUtensorMap tm_q, tm_k, tm_v;
  cudaError_t e;
  if ((e = sa_map(&tm_q, q, B, N, H)) != cudaSuccess) return e;
  if ((e = sa_map(&tm_k, k, B, N, H)) != cudaSuccess) return e;
  if ((e = sa_map(&tm_v, v, B, N, H)) != cudaSuccess) return e;
  if ((e = cudaFuncSetAttribute(sa_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem)) !=
      cudaSuccess)
    return e;
  SaParams sp{seq_lens, (__nv_bfloat16 *)o, B, H, N};
  dim3 grid((N + kQ - 1) / kQ, H, B);
  sa_kernel<<<grid, kThreads, kSmem, st>>>(sp, tm_q, tm_k, tm_v);
  count_launch();
  return cudaGetLastError();
}

unsigned sa_device_error(bool reset) {
  unsigned v = 0;
  if (cudaMemcpyFromSymbol(&v, g_sa_error, sizeof(v)) != cudaSuccess) return 0xFFFFFFFFu;
  if (reset) {
    const unsigned z = 0;
    if (cudaMemcpyToSymbol(g_sa_error, &z, sizeof(z)) != cudaSuccess) return 0xFFFFFFFFu;
  }
  return v;
}

}  // namespace gbla
