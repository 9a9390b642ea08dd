// Tensor-core tree attention (LTD section 3.2, "Draft Tree Verification";
// SpecInfer-style tree mask) for bf16 and head_dim 128 on sm_103a.
//
// Work split: a CTA owns one 128-row tile of the query rows of one KV head
// (row r = slot * G + g, so all G query heads sharing the KV head ride on
// every K/V byte) and one split of that head's keys.  Per 128-key chunk:
//   TMA (warp 0)   K and V chunks -> a 2-stage shared-memory ring, 128-byte
//                  swizzle, plus the Q tile once;
//   MMA (warp 1)   S = Q K^T into tensor memory (double-buffered), then
//                  O += P V into a tensor-memory accumulator, software-
//                  pipelined so S of chunk j+1 overlaps the softmax of j;
//   softmax (warps 4-7, one thread per row / TMEM lane)  read S, apply the
//                  prefix + ancestor-bit mask, keep a running max that only
//                  moves (rescaling O in TMEM) when it grows by more than
//                  2^8, write P as bf16 into swizzled shared memory.
// With one split the CTA normalises and writes bf16 output; otherwise it
// writes (O, max, sum) partials and a small merge kernel combines splits.
// Every mbarrier wait is bounded: on timeout the CTA flags
// LTD_DEVERR_TIMEOUT, drains its own TMA loads and MMAs, frees its tensor
// memory and returns.
#include "ltd_common.cuh"
#include "ltd_internal.h"
#include "tc_util.cuh"

namespace ltd {

namespace {

constexpr int kBM = 128;  // query rows per CTA = TMEM lanes
constexpr int kBN = 128;  // keys per chunk
constexpr int kD = 128;
constexpr int kThreads = 256;
constexpr int kMaxW32 = LTD_MAX_N / 32;
constexpr uint32_t kHalf = 16384;       // 128 rows x 128 bytes
constexpr uint32_t kTile = 2 * kHalf;   // 128 x 128 bf16
constexpr uint32_t kOffQ = 0;
constexpr uint32_t kOffK = kOffQ + kTile;
constexpr uint32_t kOffV = kOffK + 2 * kTile;
constexpr uint32_t kOffP = kOffV + 2 * kTile;
constexpr uint32_t kOffMask = kOffP + kTile;
constexpr uint32_t kOffBar = kOffMask + kBM * kMaxW32 * 4;
constexpr uint32_t kOffHolder = kOffBar + 16 * 8;
constexpr uint32_t kSmemBytes = kOffHolder + 16 + 1024;  // + alignment slack
constexpr uint32_t kTmemCols = 512;  // S0 | S1 | O (| unused)
constexpr float kRescaleThreshold = 8.f;  // log2 units

enum Bar { QFULL = 0, KFULL = 1, VFULL = 3, KVEMPTY = 5, SFULL = 7, SFREE = 9, PFULL = 11,
           PVDONE = 12, FIN = 13 };

struct TcArgs {
  int32_t batch, hq, hkv, G, n_max, s_cap, max_ctx, W32;
  int32_t splits, n_tiles;
  const int32_t* ctx;
  const int32_t* n_verify;
  const uint32_t* mask;
  float scale_log2;
  __nv_bfloat16* out;
  float4* ws_o;   // [cta][128 rows][32] float4
  float2* ws_ml;  // [cta][128] (max in log2 units, sum)
  uint32_t* err;
};

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&v);
}

__global__ void __launch_bounds__(kThreads, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tq, const __grid_constant__ CUtensorMap tk,
                   const __grid_constant__ CUtensorMap tv, const TcArgs a) {
  extern __shared__ uint8_t smem_raw[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int split = blockIdx.x, tile = blockIdx.y;
  const int b = blockIdx.z / a.hkv, kvh = blockIdx.z % a.hkv;

  const int ctx = a.ctx[b];
  const int N = a.n_verify[b];
  if (N < 1 || N > a.n_max || ctx < 0 || ctx > a.max_ctx || ctx + N > a.s_cap) {
    if (tid == 0 && split == 0 && tile == 0 && kvh == 0)
      flag_error(a.err, (N < 1 || N > a.n_max) ? LTD_DEVERR_NVERIFY : LTD_DEVERR_CTX);
    return;
  }
  const int M = N * a.G;
  if (tile * kBM >= M) return;
  const int nk = ctx + N;
  const int nch = (nk + kBN - 1) / kBN;
  const int cs = split * nch / a.splits, ce = (split + 1) * nch / a.splits;
  const int nc = ce - cs;
  const int key_lo = cs * kBN, key_hi = min(ce * kBN, nk);
  const int64_t cta = ((static_cast<int64_t>(blockIdx.z) * a.n_tiles + tile) * a.splits) + split;
  if (nc <= 0) {  // empty split: contributes nothing to the merge
    if (tid >= 128) a.ws_ml[cta * kBM + (tid - 128)] = make_float2(-CUDART_INF_F, 0.f);
    return;
  }

  const uint32_t raw = tc::smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  uint32_t* mask_s = reinterpret_cast<uint32_t*>(gbase + kOffMask);
  uint32_t* holder = reinterpret_cast<uint32_t*>(gbase + kOffHolder);
  auto bar = [&](int i) { return base + kOffBar + 8u * i; };

  if (tid == 0) {
    tc::mbar_init(bar(QFULL), 1);
    for (int s = 0; s < 2; ++s) {
      tc::mbar_init(bar(KFULL + s), 1);
      tc::mbar_init(bar(VFULL + s), 1);
      tc::mbar_init(bar(KVEMPTY + s), 1);
      tc::mbar_init(bar(SFULL + s), 1);
      tc::mbar_init(bar(SFREE + s), 128);
    }
    tc::mbar_init(bar(PFULL), 128);
    tc::mbar_init(bar(PVDONE), 1);
    tc::mbar_init(bar(FIN), 1);
    tc::mbar_init_fence();
  }
  if (warp == 1) {
    tc::tmem_alloc(tc::smem_u32(holder), kTmemCols);
    tc::tmem_relinquish();
  }
  const int i = tid - 128;  // softmax row (TMEM lane) for warps 4-7
  const int R = tile * kBM + i;
  const bool row_ok = (tid >= 128) && (R < M);
  const int slot = row_ok ? R / a.G : 0;
  if (tid >= 128) {
    for (int w = 0; w < a.W32; ++w)
      mask_s[i * kMaxW32 + w] =
          row_ok ? a.mask[(static_cast<int64_t>(b) * a.n_max + slot) * a.W32 + w] : 0u;
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = *holder;
  bool ok = true;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      int issued[2] = {0, 0};
      tc::tma_prefetch(&tq);
      tc::tma_prefetch(&tk);
      tc::tma_prefetch(&tv);
      tc::mbar_expect_tx(bar(QFULL), kTile);
      const int qrow = b * a.n_max + tile * (kBM / a.G);
      for (int h = 0; h < 2; ++h)
        tc::tma_load_3d(base + kOffQ + h * kHalf, &tq, bar(QFULL), h * 64, kvh * a.G, qrow);
      const int kvrow = b * a.hkv + kvh;
      for (int j = 0; j < nc && ok; ++j) {
        const int st = j & 1;
        if (j >= 2) ok = tc::mbar_wait(bar(KVEMPTY + st), ((j >> 1) - 1) & 1);
        if (!ok) break;
        const int key0 = key_lo + j * kBN;
        tc::mbar_expect_tx(bar(KFULL + st), kTile);
        for (int h = 0; h < 2; ++h)
          tc::tma_load_3d(base + kOffK + st * kTile + h * kHalf, &tk, bar(KFULL + st), h * 64, key0,
                          kvrow);
        tc::mbar_expect_tx(bar(VFULL + st), kTile);
        for (int h = 0; h < 2; ++h)
          tc::tma_load_3d(base + kOffV + st * kTile + h * kHalf, &tv, bar(VFULL + st), h * 64, key0,
                          kvrow);
        ++issued[st];
      }
      // drain: every load this CTA issued has landed before it can exit
      tc::mbar_wait(bar(QFULL), 0);
      for (int st = 0; st < 2; ++st)
        if (issued[st] > 0) {
          tc::mbar_wait(bar(KFULL + st), (issued[st] - 1) & 1);
          tc::mbar_wait(bar(VFULL + st), (issued[st] - 1) & 1);
        }
      if (!ok) flag_error(a.err, LTD_DEVERR_TIMEOUT);
    }
  } else if (warp == 1) {
    // ----------------------------------------------------------------- MMA
    if (lane == 0) {
      const uint32_t id_s = tc::idesc_bf16(kBM, kBN, false);
      const uint32_t id_o = tc::idesc_bf16(kBM, kD, true);
      const uint32_t t_o = tmem + 2 * kBN;
      ok = tc::mbar_wait(bar(QFULL), 0);
      for (int j = 0; j <= nc && ok; ++j) {
        if (j < nc) {
          const int st = j & 1;
          ok = tc::mbar_wait(bar(KFULL + st), (j >> 1) & 1);
          if (ok && j >= 2) ok = tc::mbar_wait(bar(SFREE + st), ((j >> 1) - 1) & 1);
          if (!ok) break;
          tc::fence_after_sync();
          for (int ks = 0; ks < 8; ++ks) {
            const uint64_t da = tc::sdesc_sw128(base + kOffQ + (ks >> 2) * kHalf + (ks & 3) * 32, 16, 1024);
            const uint64_t db =
                tc::sdesc_sw128(base + kOffK + st * kTile + (ks >> 2) * kHalf + (ks & 3) * 32, 16, 1024);
            tc::mma_bf16(tmem + st * kBN, da, db, id_s, ks > 0 ? 1u : 0u);
          }
          tc::mma_commit(bar(SFULL + st));
        }
        if (j >= 1) {
          const int jj = j - 1, st = jj & 1;
          ok = tc::mbar_wait(bar(PFULL), jj & 1);
          if (ok) ok = tc::mbar_wait(bar(VFULL + st), (jj >> 1) & 1);
          if (!ok) break;
          tc::fence_after_sync();
          for (int ks = 0; ks < 8; ++ks) {
            const uint64_t da = tc::sdesc_sw128(base + kOffP + (ks >> 2) * kHalf + (ks & 3) * 32, 16, 1024);
            const uint64_t db = tc::sdesc_sw128(base + kOffV + st * kTile + ks * 2048, kHalf, 1024);
            tc::mma_bf16(t_o, da, db, id_o, (jj > 0 || ks > 0) ? 1u : 0u);
          }
          tc::mma_commit(bar(PVDONE));
          tc::mma_commit(bar(KVEMPTY + st));
        }
      }
      // all MMAs issued by this thread complete before tensor memory is freed
      tc::mma_commit(bar(FIN));
      tc::mbar_wait(bar(FIN), 0);
      if (!ok) flag_error(a.err, LTD_DEVERR_TIMEOUT);
    }
  } else if (warp >= 4) {
    // ------------------------------------------------------------- softmax
    const uint32_t t_lane = tmem + ((32u * (warp & 3)) << 16);
    const uint32_t* mrow_bits = mask_s + i * kMaxW32;
    float m = -CUDART_INF_F, l = 0.f;
    const int vis_all_below = min(ctx, key_hi);  // keys below this are all visible
    for (int j = 0; j < nc; ++j) {
      const int sb = j & 1;
      ok = tc::mbar_wait(bar(SFULL + sb), (j >> 1) & 1);
      ok = __all_sync(0xFFFFFFFFu, ok);
      if (!ok) break;
      tc::fence_after_sync();
      float s[kBN];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        tc::Frag32 f;
        tc::tmem_ld32(t_lane + sb * kBN + 32 * q, f);
        tc::tmem_wait_ld(f);
#pragma unroll
        for (int c = 0; c < 32; ++c) s[32 * q + c] = __uint_as_float(f.r[c]);
      }
      tc::fence_before_sync();
      tc::mbar_arrive(bar(SFREE + sb));

      const int kbase = key_lo + j * kBN;
      float cmax = -CUDART_INF_F;
      if (kbase + kBN <= vis_all_below) {
#pragma unroll
        for (int c = 0; c < kBN; ++c) {
          s[c] = row_ok ? s[c] * a.scale_log2 : -CUDART_INF_F;
          cmax = fmaxf(cmax, s[c]);
        }
      } else {
#pragma unroll
        for (int c = 0; c < kBN; ++c) {
          const int kk = kbase + c;
          bool vis = row_ok && kk < key_hi;
          if (vis && kk >= ctx) {
            const int js = kk - ctx;
            vis = (mrow_bits[js >> 5] >> (js & 31)) & 1u;
          }
          s[c] = vis ? s[c] * a.scale_log2 : -CUDART_INF_F;
          cmax = fmaxf(cmax, s[c]);
        }
      }
      // P buffer and O are free once the previous chunk's P V finished
      if (j >= 1) {
        ok = tc::mbar_wait(bar(PVDONE), (j - 1) & 1);
        ok = __all_sync(0xFFFFFFFFu, ok);
        if (!ok) break;
      }
      float mnew = m;
      if (cmax > m + kRescaleThreshold || (m == -CUDART_INF_F && cmax > -CUDART_INF_F)) mnew = cmax;
      const bool need = (mnew != m) && (m != -CUDART_INF_F) && (j >= 1);
      if (__any_sync(0xFFFFFFFFu, need)) {
        const float alpha = need ? tc::ex2(m - mnew) : 1.f;
        l *= alpha;
        tc::fence_after_sync();
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          tc::Frag32 f;
          tc::tmem_ld32(t_lane + 2 * kBN + 32 * q, f);
          tc::tmem_wait_ld(f);
#pragma unroll
          for (int c = 0; c < 32; ++c) f.r[c] = __float_as_uint(__uint_as_float(f.r[c]) * alpha);
          tc::tmem_st32(t_lane + 2 * kBN + 32 * q, f);
        }
        tc::tmem_wait_st();
      }
      m = mnew;
      // P row (bf16) into the K-major 128-byte-swizzled operand tile
      uint8_t* prow = gbase + kOffP + i * 128;
      float lsum = 0.f;
#pragma unroll
      for (int c8 = 0; c8 < 16; ++c8) {
        float p[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const float t = s[8 * c8 + e];
          p[e] = (m == -CUDART_INF_F || t == -CUDART_INF_F) ? 0.f : tc::ex2(t - m);
          lsum += p[e];
        }
        uint4 w;
        w.x = pack_bf16(p[0], p[1]);
        w.y = pack_bf16(p[2], p[3]);
        w.z = pack_bf16(p[4], p[5]);
        w.w = pack_bf16(p[6], p[7]);
        const int half = c8 >> 3, cc = c8 & 7;
        *reinterpret_cast<uint4*>(prow + half * kHalf + ((cc ^ (i & 7)) << 4)) = w;
      }
      l += lsum;
      tc::fence_smem_async();
      tc::fence_before_sync();
      tc::mbar_arrive(bar(PFULL));
    }
    if (ok) {
      ok = tc::mbar_wait(bar(PVDONE), (nc - 1) & 1);
      ok = __all_sync(0xFFFFFFFFu, ok);
    }
    if (ok) {
      tc::fence_after_sync();
      const int g = row_ok ? R % a.G : 0;
      if (a.splits == 1) {
        const float inv = l > 0.f ? 1.f / l : 0.f;
        __nv_bfloat16* dst =
            a.out + ((static_cast<int64_t>(b) * a.n_max + slot) * a.hq + kvh * a.G + g) * kD;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          tc::Frag32 f;
          tc::tmem_ld32(t_lane + 2 * kBN + 32 * q, f);
          tc::tmem_wait_ld(f);
          if (row_ok) {
#pragma unroll
            for (int c = 0; c < 32; c += 8) {
              uint4 w;
              w.x = pack_bf16(__uint_as_float(f.r[c]) * inv, __uint_as_float(f.r[c + 1]) * inv);
              w.y = pack_bf16(__uint_as_float(f.r[c + 2]) * inv, __uint_as_float(f.r[c + 3]) * inv);
              w.z = pack_bf16(__uint_as_float(f.r[c + 4]) * inv, __uint_as_float(f.r[c + 5]) * inv);
              w.w = pack_bf16(__uint_as_float(f.r[c + 6]) * inv, __uint_as_float(f.r[c + 7]) * inv);
              *reinterpret_cast<uint4*>(dst + 32 * q + c) = w;
            }
          }
        }
      } else {
        float4* wo = a.ws_o + (cta * kBM + i) * 32;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          tc::Frag32 f;
          tc::tmem_ld32(t_lane + 2 * kBN + 32 * q, f);
          tc::tmem_wait_ld(f);
#pragma unroll
          for (int c4 = 0; c4 < 8; ++c4)
            wo[8 * q + c4] =
                make_float4(__uint_as_float(f.r[4 * c4]), __uint_as_float(f.r[4 * c4 + 1]),
                            __uint_as_float(f.r[4 * c4 + 2]), __uint_as_float(f.r[4 * c4 + 3]));
        }
        a.ws_ml[cta * kBM + i] = make_float2(row_ok ? m : -CUDART_INF_F, row_ok ? l : 0.f);
      }
    } else if (lane == 0) {
      flag_error(a.err, LTD_DEVERR_TIMEOUT);
    }
  }

  tc::fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, kTmemCols);
  }
}

// Combine the split partials of every row: weights 2^(m_s - max m).  One
// warp per row, lane c owns output dims 4c..4c+3, so both the partial reads
// (row-major [cta][row][32 float4]) and the bf16 output writes coalesce.
constexpr int kMergeRows = 8;

__global__ void __launch_bounds__(kMergeRows * 32) attn_tc_merge_kernel(const TcArgs a) {
  const int lane = threadIdx.x & 31;
  const int64_t grow = static_cast<int64_t>(blockIdx.x) * kMergeRows + (threadIdx.x >> 5);
  const int64_t rows_per_bh = static_cast<int64_t>(a.n_tiles) * kBM;
  const int bh = static_cast<int>(grow / rows_per_bh);
  if (bh >= a.batch * a.hkv) return;
  const int R = static_cast<int>(grow % rows_per_bh);
  const int tile = R / kBM, i = R % kBM;
  const int b = bh / a.hkv, kvh = bh % a.hkv;
  const int ctx = a.ctx[b];
  const int N = a.n_verify[b];
  if (N < 1 || N > a.n_max || ctx < 0 || ctx > a.max_ctx || ctx + N > a.s_cap) return;
  if (R >= N * a.G) return;
  const int slot = R / a.G, g = R % a.G;
  const int64_t cta0 = (static_cast<int64_t>(bh) * a.n_tiles + tile) * a.splits;
  float mx = -CUDART_INF_F;
  for (int s = 0; s < a.splits; ++s) {
    const float2 ml = a.ws_ml[(cta0 + s) * kBM + i];
    if (ml.y > 0.f) mx = fmaxf(mx, ml.x);
  }
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  float L = 0.f;
  for (int s = 0; s < a.splits; ++s) {
    const float2 ml = a.ws_ml[(cta0 + s) * kBM + i];
    if (!(ml.y > 0.f)) continue;
    const float w = tc::ex2(ml.x - mx);
    L += w * ml.y;
    const float4 v = a.ws_o[((cta0 + s) * kBM + i) * 32 + lane];
    acc.x += w * v.x;
    acc.y += w * v.y;
    acc.z += w * v.z;
    acc.w += w * v.w;
  }
  const float inv = L > 0.f ? 1.f / L : 0.f;
  __nv_bfloat16* dst =
      a.out + ((static_cast<int64_t>(b) * a.n_max + slot) * a.hq + kvh * a.G + g) * kD + 4 * lane;
  uint2 w2;
  w2.x = pack_bf16(acc.x * inv, acc.y * inv);
  w2.y = pack_bf16(acc.z * inv, acc.w * inv);
  *reinterpret_cast<uint2*>(dst) = w2;
}

struct Plan {
  int n_tiles, splits;
};

Plan plan(int32_t batch, int32_t hq, int32_t hkv, int32_t n_max, int32_t max_ctx) {
  const int G = hq / hkv;
  Plan p{};
  p.n_tiles = (n_max * G + kBM - 1) / kBM;
  const int64_t base = static_cast<int64_t>(batch) * hkv * p.n_tiles;
  const int nch = (max_ctx + n_max + kBN - 1) / kBN;
  constexpr int64_t kSMs = 152;
  int s = base >= kSMs ? 1 : static_cast<int>(kSMs / base);
  s = s < 1 ? 1 : s;
  s = s > nch ? nch : s;
  p.splits = s;
  return p;
}

using EncodeFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                              const cuuint64_t*, const cuuint32_t*, const cuuint32_t*,
                              CUtensorMapInterleave, CUtensorMapSwizzle, CUtensorMapL2promotion,
                              CUtensorMapFloatOOBfill);

EncodeFn encode_fn() {
  static EncodeFn fn = nullptr;
  static bool tried = false;
  if (!tried) {
    tried = true;
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeFn>(p);
  }
  return fn;
}

}  // namespace

bool encode_tmap_bf16_3d(CUtensorMap* map, const void* base, uint64_t d0, uint64_t d1, uint64_t d2,
                         uint64_t stride1, uint64_t stride2, uint32_t b0, uint32_t b1, uint32_t b2) {
  EncodeFn fn = encode_fn();
  if (fn == nullptr) return false;
  const cuuint64_t dims[3] = {d0, d1, d2};
  const cuuint64_t strides[2] = {stride1, stride2};
  const cuuint32_t box[3] = {b0, b1, b2};
  const cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool attn_tc_supported(const AttnParams& p, ltd_dtype dtype) {
  if (dtype != LTD_BF16 || p.d != kD || p.hkv < 1 || p.hq % p.hkv != 0) return false;
  const int G = p.hq / p.hkv;
  return G >= 1 && G <= kBM && kBM % G == 0 && p.n_max <= LTD_MAX_N;
}

size_t attn_tc_workspace(int32_t batch, int32_t hq, int32_t hkv, int32_t d, int32_t n_max,
                         int32_t max_ctx) {
  (void)d;
  const Plan pl = plan(batch, hq, hkv, n_max, max_ctx);
  if (pl.splits == 1) return 0;
  const size_t ctas = static_cast<size_t>(batch) * hkv * pl.n_tiles * pl.splits;
  return ctas * (32 * kBM * sizeof(float4) + kBM * sizeof(float2));
}

int32_t attn_tc_launches(int32_t batch, int32_t hq, int32_t hkv, int32_t n_max, int32_t max_ctx) {
  return plan(batch, hq, hkv, n_max, max_ctx).splits > 1 ? 2 : 1;
}

cudaError_t launch_attn_tc(const AttnParams& p, cudaStream_t s) {
  const Plan pl = plan(p.batch, p.hq, p.hkv, p.n_max, p.max_ctx);
  TcArgs a{};
  a.batch = p.batch;
  a.hq = p.hq;
  a.hkv = p.hkv;
  a.G = p.hq / p.hkv;
  a.n_max = p.n_max;
  a.s_cap = p.s_cap;
  a.max_ctx = p.max_ctx;
  a.W32 = (p.n_max + 31) / 32;
  a.splits = pl.splits;
  a.n_tiles = pl.n_tiles;
  a.ctx = p.ctx;
  a.n_verify = p.n_verify;
  a.mask = p.mask;
  a.scale_log2 = p.scale * 1.4426950408889634f;
  a.out = static_cast<__nv_bfloat16*>(p.out);
  const size_t ctas = static_cast<size_t>(p.batch) * p.hkv * pl.n_tiles * pl.splits;
  a.ws_o = static_cast<float4*>(p.ws);
  a.ws_ml = reinterpret_cast<float2*>(static_cast<char*>(p.ws) + ctas * 32 * kBM * sizeof(float4));
  a.err = p.err;
  if (pl.splits > 1 && p.ws_bytes < attn_tc_workspace(p.batch, p.hq, p.hkv, p.d, p.n_max, p.max_ctx))
    return cudaErrorInvalidValue;

  CUtensorMap tq, tk, tv;
  const uint64_t row = kD * 2;
  if (!encode_tmap_bf16_3d(&tq, p.q, kD, p.hq, static_cast<uint64_t>(p.batch) * p.n_max, row,
                           row * p.hq, 64, a.G, kBM / a.G))
    return cudaErrorInvalidValue;
  if (!encode_tmap_bf16_3d(&tk, p.k, kD, p.s_cap, static_cast<uint64_t>(p.batch) * p.hkv, row,
                           row * p.s_cap, 64, kBN, 1))
    return cudaErrorInvalidValue;
  if (!encode_tmap_bf16_3d(&tv, p.v, kD, p.s_cap, static_cast<uint64_t>(p.batch) * p.hkv, row,
                           row * p.s_cap, 64, kBN, 1))
    return cudaErrorInvalidValue;
  cudaError_t e = cudaFuncSetAttribute(attn_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(kSmemBytes));
  if (e != cudaSuccess) return e;
  const dim3 grid(pl.splits, pl.n_tiles, p.batch * p.hkv);
  attn_tc_kernel<<<grid, kThreads, kSmemBytes, s>>>(tq, tk, tv, a);
  e = cudaGetLastError();
  if (e != cudaSuccess || pl.splits == 1) return e;
  const int64_t rows = static_cast<int64_t>(p.batch) * p.hkv * pl.n_tiles * kBM;
  attn_tc_merge_kernel<<<static_cast<unsigned>((rows + kMergeRows - 1) / kMergeRows),
                         kMergeRows * 32, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace ltd
