// Tensor-core tree attention (LTD section 3.2, "Draft Tree Verification";
// SpecInfer-style tree mask) for bf16 and head_dim 128 on sm_103a.
//
// Work split: a CTA owns two 128-row tiles ("a" and "b") of the query rows
// of one KV head (row r = slot * G + g, so the G query heads of a KV head
// share every K/V byte) and one split of that head's keys; the splits of one
// (sequence, head, tile pair) form a thread-block cluster of up to 16 CTAs.
//   warp 0      TMA: both Q tiles once, then 128-key K and V chunks into
//               two-stage rings (128-byte swizzle);
//   warp 1      tcgen05.mma: S_x = Q_x K^T into tensor memory, then
//               O_x += P_x V with P_x read from tensor memory; the order
//               PV_a(j), S_a(j+1), PV_b(j), S_b(j+1) lets one tile's
//               softmax run while the tensor core works on the other;
//   warps 4-7   softmax of tile a, warps 8-11 of tile b, one thread per row
//               (= tensor-memory lane): read S, apply the prefix + ancestor
//               mask, keep a running max that rescales O only when it grows
//               by more than 2^8, write P as bf16 over S's columns.
// Tensor memory (512 columns): S_a | S_b | O_a | O_b.
// After the last MMA every CTA stages its rows as O/l in bf16 plus the
// log-sum-exp, and (after one cluster barrier) bulk-copies each block of
// rows to the cluster CTA that owns them through distributed shared memory;
// each CTA then combines its rows across all splits locally and writes bf16
// output.  No global workspace, no second kernel.
// Every mbarrier wait is bounded: on timeout the CTA flags
// LTD_DEVERR_TIMEOUT, drains its own TMA loads and MMAs, and still joins
// the cluster barrier and sends every block its peers expect (so no peer
// waits on it forever), frees its tensor memory and returns.
#include <mutex>

#include "ltd_common.cuh"
#include "ltd_internal.h"
#include "tc_util.cuh"

namespace ltd {

namespace {

constexpr int kBM = 128;  // rows per tile = TMEM lanes
constexpr int kBN = 128;  // keys per chunk
constexpr int kD = 128;
constexpr int kRows = 2 * kBM;
constexpr int kThreads = 384;
constexpr int kWarps = kThreads / 32;
constexpr int kMaxW32 = LTD_MAX_N / 32;
constexpr int kMaxCluster = 16;
constexpr uint32_t kHalf = 16384;      // 128 rows x 128 bytes
constexpr uint32_t kTile = 2 * kHalf;  // 128 x 128 bf16
constexpr uint32_t kOffQ = 0;                        // Q_a, Q_b
constexpr uint32_t kOffK = kOffQ + 2 * kTile;        // two stages
constexpr uint32_t kOffV = kOffK + 2 * kTile;        // two stages
constexpr uint32_t kOffMask = kOffV + 2 * kTile;     // [256][8] words
constexpr uint32_t kOffBar = kOffMask + kRows * kMaxW32 * 4;
constexpr uint32_t kOffHolder = kOffBar + 32 * 8;
constexpr uint32_t kSmemBytes = kOffHolder + 16 + 1024;  // + alignment slack
// Split reduction, over the Q/K/V space once the MMAs have finished.  CTA r
// of the cluster owns rows [r R, r R + R), R = ceil(256 / splits) rounded up
// to a multiple of 4, and receives every split's normalised O (bf16, 256
// bytes per row, 16-byte chunks swizzled by row) and log-sum-exp for them.
constexpr uint32_t kRowBytes = kD * 2;
constexpr uint32_t kOffRecvO = 0;                           // [split][R] rows, <= 80 KB
constexpr uint32_t kOffRecvL = 80 * 1024;                   // [split][R] float, <= 2 KB
constexpr uint32_t kOffStgO = 96 * 1024;                    // [256] rows
constexpr uint32_t kOffStgL = kOffStgO + kRows * kRowBytes;  // [256] float
constexpr uint32_t kTmemCols = 512;
constexpr float kRescaleThreshold = 8.f;  // log2 units

static_assert(kOffStgL + kRows * 4 <= kOffMask, "reduction buffers overlap the mask");

enum Bar { QFULL = 0, KFULL = 1, VFULL = 3, KEMPTY = 5, VEMPTY = 7, SFULL = 9, PFULL = 11, FIN = 13,
           RECV = 14 };

// Optional phase timestamps for performance work (off in normal builds).
#ifdef LTD_TRACE
__device__ unsigned long long g_attn_trace[2048][24];
#define TRACE(slot)                                                                           \
  do {                                                                                        \
    const int cta_ = blockIdx.x + gridDim.x * (blockIdx.y + gridDim.y * blockIdx.z);          \
    if (cta_ < 2048) g_attn_trace[cta_][slot] = tc::globaltimer();                            \
  } while (0)
#else
#define TRACE(slot) \
  do {              \
  } while (0)
#endif

struct TcArgs {
  int32_t batch, hq, hkv, G, n_max, s_cap, max_ctx, W32;
  int32_t splits, n_pairs;
  const int32_t* ctx;
  const int32_t* n_verify;
  const uint32_t* mask;
  float scale_log2;
  __nv_bfloat16* out;
  uint32_t* err;
};

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&v);
}

// Visibility of keys kk0 .. kk0+31 for one row as a 32-bit mask: keys below
// ctx are the prefix (always visible), key ctx + j is verified slot j (bit j
// of the row's ancestor mask), keys from key_hi on are outside this split.
__device__ __forceinline__ uint32_t low_bits(int n) {
  return n <= 0 ? 0u : (n >= 32 ? 0xFFFFFFFFu : ((1u << n) - 1u));
}
__device__ __forceinline__ uint32_t visible32(int kk0, int ctx, int key_hi, int W32,
                                              const uint32_t* mbits) {
  const uint32_t in_range = low_bits(key_hi - kk0);
  const uint32_t prefix = low_bits(ctx - kk0);
  uint32_t tree = 0u;
  const int js0 = kk0 - ctx;  // slot of bit 0 of the window (may be negative)
  if (js0 > -32 && js0 < 32 * W32) {
    const int w = js0 >> 5;  // floor division
    const int sh = js0 & 31;
    const uint32_t lo = (w >= 0 && w < W32) ? mbits[w] : 0u;
    const uint32_t hi = (w + 1 >= 0 && w + 1 < W32) ? mbits[w + 1] : 0u;
    tree = __funnelshift_r(lo, hi, sh);
  }
  return in_range & (prefix | tree);
}

__global__ void __launch_bounds__(kThreads, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tq, const __grid_constant__ CUtensorMap tk,
                   const __grid_constant__ CUtensorMap tv, const TcArgs a) {
  extern __shared__ uint8_t smem_raw[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) TRACE(0);
  const int split = blockIdx.x, pair = blockIdx.y;
  const int b = blockIdx.z / a.hkv, kvh = blockIdx.z % a.hkv;

  // Everything a CTA returns early on is shared by its whole cluster (same
  // sequence, head and tile pair), so clusters return as a unit.
  const int ctx = a.ctx[b];
  const int N = a.n_verify[b];
  if (N < 1 || N > a.n_max || ctx < 0 || ctx > a.max_ctx || ctx + N > a.s_cap) {
    if (tid == 0 && split == 0 && pair == 0 && kvh == 0)
      flag_error(a.err, (N < 1 || N > a.n_max) ? LTD_DEVERR_NVERIFY : LTD_DEVERR_CTX);
    return;
  }
  const int M = N * a.G;
  const int row0 = pair * kRows;
  if (row0 >= M) return;
  const bool has_b = row0 + kBM < M;
  const int nk = ctx + N;
  const int nch = (nk + kBN - 1) / kBN;
  const int cs = split * nch / a.splits, ce = (split + 1) * nch / a.splits;
  const int nc = ce - cs;
  const int key_lo = cs * kBN, key_hi = min(ce * kBN, nk);

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
      tc::mbar_init(bar(KEMPTY + s), 1);
      tc::mbar_init(bar(VEMPTY + s), 1);
      tc::mbar_init(bar(SFULL + s), 1);
      tc::mbar_init(bar(PFULL + s), 128);
    }
    tc::mbar_init(bar(FIN), 1);
    tc::mbar_init(bar(RECV), 1);
    tc::mbar_init_fence();
  }
  if (warp == 1) {
    tc::tmem_alloc(tc::smem_u32(holder), kTmemCols);
    tc::tmem_relinquish();
  }
  // softmax threads: tile x, TMEM lane rr % 128, staging row rr
  const int rr = tid - 128;
  const int x = rr >> 7;
  const int R = row0 + rr;
  const bool row_ok = tid >= 128 && R < M;
  if (tid >= 128) {
    const int slot = row_ok ? R / a.G : 0;
    for (int w = 0; w < a.W32; ++w)
      mask_s[rr * kMaxW32 + w] =
          row_ok ? a.mask[(static_cast<int64_t>(b) * a.n_max + slot) * a.W32 + w] : 0u;
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = *holder;
  if (tid == 0) TRACE(1);
  bool ok = true;
  const bool tile_active = tid >= 128 && (x == 0 || has_b) && nc > 0;
  float m = -CUDART_INF_F, l = 0.f;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0 && nc > 0) {
      int nk_issued[2] = {0, 0}, nv_issued[2] = {0, 0};
      tc::tma_prefetch(&tq);
      tc::tma_prefetch(&tk);
      tc::tma_prefetch(&tv);
      tc::mbar_expect_tx(bar(QFULL), has_b ? 2 * kTile : kTile);
      for (int t = 0; t < (has_b ? 2 : 1); ++t) {
        const int qrow = b * a.n_max + (row0 + t * kBM) / a.G;
        for (int h = 0; h < 2; ++h)
          tc::tma_load_3d(base + kOffQ + t * kTile + h * kHalf, &tq, bar(QFULL), h * 64, kvh * a.G,
                          qrow);
      }
      const int kvrow = b * a.hkv + kvh;
      for (int j = 0; j < nc && ok; ++j) {
        const int st = j & 1;
        const int key0 = key_lo + j * kBN;
        if (j >= 2) ok = tc::mbar_wait(bar(KEMPTY + st), ((j >> 1) - 1) & 1);
        if (!ok) break;
        tc::mbar_expect_tx(bar(KFULL + st), kTile);
        for (int h = 0; h < 2; ++h)
          tc::tma_load_3d(base + kOffK + st * kTile + h * kHalf, &tk, bar(KFULL + st), h * 64, key0,
                          kvrow);
        ++nk_issued[st];
        if (j >= 2) ok = tc::mbar_wait(bar(VEMPTY + st), ((j >> 1) - 1) & 1);
        if (!ok) break;
        tc::mbar_expect_tx(bar(VFULL + st), kTile);
        for (int h = 0; h < 2; ++h)
          tc::tma_load_3d(base + kOffV + st * kTile + h * kHalf, &tv, bar(VFULL + st), h * 64, key0,
                          kvrow);
        ++nv_issued[st];
      }
      // drain: every load this CTA issued has landed before shared memory is reused
      tc::mbar_wait(bar(QFULL), 0);
      for (int st = 0; st < 2; ++st) {
        if (nk_issued[st] > 0) tc::mbar_wait(bar(KFULL + st), (nk_issued[st] - 1) & 1);
        if (nv_issued[st] > 0) tc::mbar_wait(bar(VFULL + st), (nv_issued[st] - 1) & 1);
      }
      if (!ok) flag_error(a.err, LTD_DEVERR_TIMEOUT);
    }
  } else if (warp == 1) {
    // ----------------------------------------------------------------- MMA
    if (lane == 0 && nc > 0) {
      const uint32_t id_s = tc::idesc_bf16(kBM, kBN, false);
      const uint32_t id_o = tc::idesc_bf16(kBM, kD, true);
      const int ntile = has_b ? 2 : 1;
      auto issue_s = [&](int t, int st) {
        for (int ks = 0; ks < 8; ++ks) {
          const uint64_t da =
              tc::sdesc_sw128(base + kOffQ + t * kTile + (ks >> 2) * kHalf + (ks & 3) * 32, 16, 1024);
          const uint64_t db =
              tc::sdesc_sw128(base + kOffK + st * kTile + (ks >> 2) * kHalf + (ks & 3) * 32, 16, 1024);
          tc::mma_bf16(tmem + t * kBN, da, db, id_s, ks > 0 ? 1u : 0u);
        }
      };
      auto issue_pv = [&](int t, int st, bool acc) {
        for (int ks = 0; ks < 8; ++ks) {
          const uint64_t db = tc::sdesc_sw128(base + kOffV + st * kTile + ks * 2048, kHalf, 1024);
          tc::mma_bf16_ts(tmem + 2 * kBN + t * kD, tmem + t * kBN + 8 * ks, db, id_o,
                          (acc || ks > 0) ? 1u : 0u);
        }
      };
      ok = tc::mbar_wait(bar(QFULL), 0);
      TRACE(2);
      if (ok) ok = tc::mbar_wait(bar(KFULL + 0), 0);
      if (ok) {
        tc::fence_after_sync();
        for (int t = 0; t < ntile; ++t) {
          issue_s(t, 0);
          tc::mma_commit(bar(SFULL + t));
        }
        tc::mma_commit(bar(KEMPTY + 0));
      }
      for (int j = 0; j < nc && ok; ++j) {
        const int st = j & 1;
        const bool nxt = j + 1 < nc;
        ok = tc::mbar_wait(bar(VFULL + st), (j >> 1) & 1);
        if (ok && nxt) ok = tc::mbar_wait(bar(KFULL + ((j + 1) & 1)), ((j + 1) >> 1) & 1);
        for (int t = 0; t < ntile && ok; ++t) {
          ok = tc::mbar_wait(bar(PFULL + t), j & 1);
          if (!ok) break;
          tc::fence_after_sync();
          issue_pv(t, st, j > 0);
          if (nxt) {
            issue_s(t, (j + 1) & 1);
            tc::mma_commit(bar(SFULL + t));
          }
        }
        if (!ok) break;
        if (nxt) tc::mma_commit(bar(KEMPTY + ((j + 1) & 1)));
        tc::mma_commit(bar(VEMPTY + st));
      }
      // every MMA of this CTA completes before tensor memory is read or freed
      tc::mma_commit(bar(FIN));
      tc::mbar_wait(bar(FIN), 0);
      if (!ok) flag_error(a.err, LTD_DEVERR_TIMEOUT);
    }
  } else if (warp >= 4 && tile_active) {
    // ------------------------------------------------------------- softmax
    const uint32_t lane_off = (32u * (warp & 3)) << 16;
    const uint32_t t_s = tmem + x * kBN + lane_off;
    const uint32_t t_o = tmem + 2 * kBN + x * kD + lane_off;
    const uint32_t* mbits = mask_s + rr * kMaxW32;
    const int vis_all_below = min(ctx, key_hi);  // keys below this are all visible
    const float sl2 = a.scale_log2;
    const int w32 = a.W32;
    for (int j = 0; j < nc; ++j) {
      ok = tc::mbar_wait(bar(SFULL + x), j & 1);
      ok = __all_sync(0xFFFFFFFFu, ok);
      if (tid == 128 && j == 0) TRACE(11);

      if (!ok) break;
      tc::fence_after_sync();
      const int kbase = key_lo + j * kBN;
      const bool all_vis = kbase + kBN <= vis_all_below;
      auto vis_of = [=](int q) {
        return !row_ok ? 0u
                       : (all_vis ? 0xFFFFFFFFu
                                  : visible32(kbase + 32 * q, ctx, key_hi, w32, mbits));
      };
      // pass 1: the chunk's row max, 32 columns at a time, without branches
      // per element; on fully visible fragments the max is taken on the raw
      // scores (the scale is positive) and scaled once
      float cm[4] = {-CUDART_INF_F, -CUDART_INF_F, -CUDART_INF_F, -CUDART_INF_F};
#pragma unroll 1
      for (int q = 0; q < 4; ++q) {
        tc::Frag32 f;
        tc::tmem_ld32(t_s + 32 * q, f);
        const uint32_t vq = vis_of(q);
        tc::tmem_wait_ld(f);
        if (tid == 128 && j == 0 && q < 2) TRACE(3 + 2 * q);
        if (vq == 0xFFFFFFFFu) {
          float r[4] = {-CUDART_INF_F, -CUDART_INF_F, -CUDART_INF_F, -CUDART_INF_F};
#pragma unroll
          for (int c = 0; c < 32; ++c) r[c & 3] = fmaxf(r[c & 3], __uint_as_float(f.r[c]));
#pragma unroll
          for (int u = 0; u < 4; ++u) cm[u] = fmaxf(cm[u], r[u] * sl2);
        } else {
#pragma unroll
          for (int c = 0; c < 32; ++c) {
            const float t = ((vq >> c) & 1u) ? __uint_as_float(f.r[c]) * sl2 : -CUDART_INF_F;
            cm[c & 3] = fmaxf(cm[c & 3], t);
          }
        }
        if (tid == 128 && j == 0 && q < 2) TRACE(4 + 2 * q);
      }
      const float cmax = fmaxf(fmaxf(cm[0], cm[1]), fmaxf(cm[2], cm[3]));
      if (tid == 128 && j == 0) TRACE(14);
      // S(j) complete implies P_x(j-1) V finished, so O_x is stable here
      float mnew = m;
      if (cmax > m + kRescaleThreshold || (m == -CUDART_INF_F && cmax > -CUDART_INF_F)) mnew = cmax;
      const bool need = (mnew != m) && (m != -CUDART_INF_F) && (j >= 1);
      if (__any_sync(0xFFFFFFFFu, need)) {
        const float alpha = need ? tc::ex2(m - mnew) : 1.f;
        l *= alpha;
#pragma unroll 1
        for (int q = 0; q < 4; ++q) {
          tc::Frag32 f;
          tc::tmem_ld32(t_o + 32 * q, f);
          tc::tmem_wait_ld(f);
#pragma unroll
          for (int c = 0; c < 32; ++c) f.r[c] = __float_as_uint(__uint_as_float(f.r[c]) * alpha);
          tc::tmem_st32(t_o + 32 * q, f);
        }
      }
      m = mnew;
      // pass 2: P = 2^(score - m) as bf16 pairs; fragment q (columns
      // 32q..32q+31) becomes P columns 16q..16q+15, all already read
      float2 ls2[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
      const float mz = (m == -CUDART_INF_F) ? 0.f : m;  // m = -inf only if all are hidden
      const float2 sl22 = make_float2(sl2, sl2), nm2 = make_float2(-mz, -mz);
#pragma unroll 1
      for (int q = 0; q < 4; ++q) {
        tc::Frag32 f;
        tc::tmem_ld32(t_s + 32 * q, f);
        const uint32_t vq = vis_of(q);
        tc::tmem_wait_ld(f);
        tc::Frag16 pf;
        if (vq == 0xFFFFFFFFu) {
#pragma unroll
          for (int c = 0; c < 16; ++c) {
            const float2 t = __ffma2_rn(
                make_float2(__uint_as_float(f.r[2 * c]), __uint_as_float(f.r[2 * c + 1])), sl22, nm2);
            const float2 pp = make_float2(tc::ex2(t.x), tc::ex2(t.y));
            ls2[c & 1] = __fadd2_rn(ls2[c & 1], pp);
            pf.r[c] = pack_bf16(pp.x, pp.y);
          }
        } else {
#pragma unroll
          for (int c = 0; c < 16; ++c) {
            const float t0 =
                ((vq >> (2 * c)) & 1u) ? __uint_as_float(f.r[2 * c]) * sl2 : -CUDART_INF_F;
            const float t1 =
                ((vq >> (2 * c + 1)) & 1u) ? __uint_as_float(f.r[2 * c + 1]) * sl2 : -CUDART_INF_F;
            const float2 pp = make_float2(tc::ex2(t0 - mz), tc::ex2(t1 - mz));
            ls2[c & 1] = __fadd2_rn(ls2[c & 1], pp);
            pf.r[c] = pack_bf16(pp.x, pp.y);
          }
        }
        tc::tmem_st16(t_s + 16 * q, pf);
      }
      const float2 lsum = __fadd2_rn(ls2[0], ls2[1]);
      l += lsum.x + lsum.y;
      if (tid == 128 && j == 0) TRACE(15);
      tc::tmem_wait_st();
      tc::fence_before_sync();
      tc::mbar_arrive(bar(PFULL + x));
      if (tid == 128 && j == 0) TRACE(12);
    }
    if (tid == 128) TRACE(13);
    if (ok) {
      ok = tc::mbar_wait(bar(FIN), 0);
      ok = __all_sync(0xFFFFFFFFu, ok);
    }
    if (!ok && lane == 0) flag_error(a.err, LTD_DEVERR_TIMEOUT);
  }

  // --------------------- exchange partials with the cluster (bulk DSMEM)
  tc::fence_before_sync();
  __syncthreads();
  if (tid == 0) TRACE(16);
  const int S = a.splits;
  const int rank = static_cast<int>(tc::cluster_rank());
  const int R4 = (((kRows + S - 1) / S) + 3) & ~3;
  const int n_own = max(0, min(R4, kRows - rank * R4));
  if (tid == 0) tc::mbar_expect_tx(bar(RECV), static_cast<uint32_t>(S * n_own) * (kRowBytes + 4));
  // stage this split's rows: O / l in bf16 and lse = m + log2(l)
  if (tid >= 128) {
    float lse = -CUDART_INF_F;
    uint8_t* srow = gbase + kOffStgO + rr * kRowBytes;
    if (tile_active && ok) {
      tc::fence_after_sync();
      const uint32_t t_o = tmem + 2 * kBN + x * kD + ((32u * (warp & 3)) << 16);
      const float inv = l > 0.f ? 1.f / l : 0.f;
#pragma unroll 1
      for (int q = 0; q < 4; ++q) {
        tc::Frag32 f;
        tc::tmem_ld32(t_o + 32 * q, f);
        tc::tmem_wait_ld(f);
#pragma unroll
        for (int c16 = 0; c16 < 4; ++c16) {
          const int c = 4 * q + c16;  // 16-byte chunk (8 values) of the row
          uint4 w;
          w.x = pack_bf16(__uint_as_float(f.r[8 * c16]) * inv, __uint_as_float(f.r[8 * c16 + 1]) * inv);
          w.y = pack_bf16(__uint_as_float(f.r[8 * c16 + 2]) * inv, __uint_as_float(f.r[8 * c16 + 3]) * inv);
          w.z = pack_bf16(__uint_as_float(f.r[8 * c16 + 4]) * inv, __uint_as_float(f.r[8 * c16 + 5]) * inv);
          w.w = pack_bf16(__uint_as_float(f.r[8 * c16 + 6]) * inv, __uint_as_float(f.r[8 * c16 + 7]) * inv);
          *reinterpret_cast<uint4*>(srow + ((c ^ (rr & 15)) << 4)) = w;
        }
      }
      if (row_ok && l > 0.f) lse = m + __log2f(l);
    }
    reinterpret_cast<float*>(gbase + kOffStgL)[rr] = lse;
    tc::fence_smem_async();  // staging becomes visible to the bulk copies
  }
  __syncthreads();
  // every CTA has registered its receive count and is past its last MMA and
  // TMA load, so its ring buffers can now be written by peers
  tc::cluster_sync();
  if (tid == 0) TRACE(7);
  if (tid == 0) {
    for (int r = 0; r < S; ++r) {
      const int n = max(0, min(R4, kRows - r * R4));
      if (n == 0) continue;
      const uint32_t pbar = tc::mapa(bar(RECV), r);
      tc::bulk_s2cluster(tc::mapa(base + kOffRecvO + (rank * R4) * kRowBytes, r),
                         base + kOffStgO + (r * R4) * kRowBytes, n * kRowBytes, pbar);
      tc::bulk_s2cluster(tc::mapa(base + kOffRecvL + (rank * R4) * 4, r),
                         base + kOffStgL + (r * R4) * 4, n * 4, pbar);
    }
    tc::bulk_commit();
  }
  const bool got = tc::mbar_wait(bar(RECV), 0);
  if (!got && tid == 0) flag_error(a.err, LTD_DEVERR_TIMEOUT);
  if (tid == 0) TRACE(8);

  // ------------------------- combine the splits of this CTA's rows (local)
  if (got) {
    const uint8_t* recv_o = gbase + kOffRecvO;
    const float* recv_l = reinterpret_cast<const float*>(gbase + kOffRecvL);
    const int ch = lane >> 1, half = lane & 1;  // lane owns output dims 4 lane .. 4 lane + 3
    for (int lr = warp; lr < n_own; lr += kWarps) {
      const int r = rank * R4 + lr;
      const int Rr = row0 + r;
      if (Rr >= M) continue;
      const uint32_t coff = (((ch ^ (r & 15)) << 4) + half * 8);
      float lp[kMaxCluster];
      uint2 vp[kMaxCluster];
#pragma unroll
      for (int p = 0; p < kMaxCluster; ++p) {
        if (p < S) {
          lp[p] = recv_l[p * R4 + lr];
          vp[p] = *reinterpret_cast<const uint2*>(recv_o + (p * R4 + lr) * kRowBytes + coff);
        }
      }
      float mx = -CUDART_INF_F;
#pragma unroll
      for (int p = 0; p < kMaxCluster; ++p)
        if (p < S) mx = fmaxf(mx, lp[p]);
      float acc[4] = {0.f, 0.f, 0.f, 0.f};
      float L = 0.f;
#pragma unroll
      for (int p = 0; p < kMaxCluster; ++p) {
        if (p < S && lp[p] > -CUDART_INF_F) {
          const float w = tc::ex2(lp[p] - mx);
          L += w;
          acc[0] += w * __uint_as_float(vp[p].x << 16);
          acc[1] += w * __uint_as_float(vp[p].x & 0xFFFF0000u);
          acc[2] += w * __uint_as_float(vp[p].y << 16);
          acc[3] += w * __uint_as_float(vp[p].y & 0xFFFF0000u);
        }
      }
      const float inv = L > 0.f ? 1.f / L : 0.f;
      const int slot = Rr / a.G, g = Rr % a.G;
      __nv_bfloat16* dst = a.out +
                           ((static_cast<int64_t>(b) * a.n_max + slot) * a.hq + kvh * a.G + g) * kD +
                           4 * lane;
      uint2 w2;
      w2.x = pack_bf16(acc[0] * inv, acc[1] * inv);
      w2.y = pack_bf16(acc[2] * inv, acc[3] * inv);
      *reinterpret_cast<uint2*>(dst) = w2;
    }
  }
  if (tid == 0) TRACE(9);
  // the sources of this CTA's outgoing copies stay valid until read
  if (tid == 0) tc::bulk_wait_read();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, kTmemCols);
  }
}

struct Plan {
  int n_pairs, splits;
};

Plan plan(int32_t batch, int32_t hq, int32_t hkv, int32_t n_max, int32_t max_ctx) {
  const int G = hq / hkv;
  Plan p{};
  p.n_pairs = (n_max * G + kRows - 1) / kRows;
  const int64_t units = static_cast<int64_t>(batch) * hkv * p.n_pairs;
  const int nch = (max_ctx + n_max + kBN - 1) / kBN;
  constexpr int64_t kSMs = 152;
  int s = units >= kSMs ? 1 : static_cast<int>(kSMs / units);
  s = s > kMaxCluster ? kMaxCluster : s;
  s = s > nch ? nch : s;
  p.splits = s < 1 ? 1 : s;
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

// Cluster size for `units` independent clusters: the largest s <= want for
// which the device can keep all of them resident at once (one wave), else
// the largest s it can run at all.  Asked once per device and size.
int max_active_clusters(int s) {
  static std::mutex mu;
  static int known[128][kMaxCluster + 1];
  static bool init = false;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 128) return 0;
  std::lock_guard<std::mutex> lock(mu);
  if (!init) {
    for (auto& row : known)
      for (int& v : row) v = -1;
    init = true;
  }
  if (known[dev][s] < 0) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(s, 1, 1);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = kSmemBytes;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = s;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    const cudaError_t e = cudaOccupancyMaxActiveClusters(&n, attn_tc_kernel, &cfg);
    if (e != cudaSuccess) {
      (void)cudaGetLastError();
      n = 0;
    }
    known[dev][s] = n;
  }
  return known[dev][s];
}

int fit_splits(int want, int64_t units) {
  for (int s = want; s > 1; --s)
    if (max_active_clusters(s) >= units) return s;
  for (int s = want; s > 1; --s)
    if (max_active_clusters(s) > 0) return s;
  return 1;
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

size_t attn_tc_workspace(int32_t, int32_t, int32_t, int32_t, int32_t, int32_t) { return 0; }

int32_t attn_tc_launches(int32_t, int32_t, int32_t, int32_t, int32_t) { return 1; }

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
  a.n_pairs = pl.n_pairs;
  a.ctx = p.ctx;
  a.n_verify = p.n_verify;
  a.mask = p.mask;
  a.scale_log2 = p.scale * 1.4426950408889634f;
  a.out = static_cast<__nv_bfloat16*>(p.out);
  a.err = p.err;

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
  e = cudaFuncSetAttribute(attn_tc_kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e != cudaSuccess) return e;

  const int splits =
      fit_splits(pl.splits, static_cast<int64_t>(p.batch) * p.hkv * pl.n_pairs);
  a.splits = splits;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(splits, pl.n_pairs, p.batch * p.hkv);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = kSmemBytes;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = splits;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, attn_tc_kernel, tq, tk, tv, a);
}

}  // namespace ltd

#ifdef LTD_TRACE
extern "C" int ltd_attn_trace_read(unsigned long long* host, int n) {
  return cudaMemcpyFromSymbol(host, ltd::g_attn_trace, sizeof(unsigned long long) * n) == cudaSuccess
             ? 0
             : 1;
}
#endif
