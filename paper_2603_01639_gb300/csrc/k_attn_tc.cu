// Tensor-core tree attention (LTD section 3.2, "Draft Tree Verification";
// SpecInfer-style tree mask) for bf16 and head_dim 128 on sm_103a.
//
// Work unit: two 128-row tiles ("a" and "b") of the query rows of one KV
// head of one sequence (row r = slot * G + g, so the G query heads of a KV
// head share every K/V byte), over one split of that head's keys.
//   warp 0      TMA: both Q tiles, then 128-key K and V chunks into
//               two-stage rings (128-byte swizzle); the first two stages are
//               issued before the setup barrier;
//   warp 1      tcgen05.mma: S_x = Q_x K^T into tensor memory, then
//               O_x += P_x V with P_x read from tensor memory; the order
//               PV_a(j), S_a(j+1), PV_b(j), S_b(j+1) lets one tile's
//               softmax run while the tensor core works on the other;
//   warps 4-7   softmax of tile a, warps 8-11 of tile b, one thread per row
//               (= tensor-memory lane) with the row's 128 scores in
//               registers: the prefix + ancestor mask, then P = 2^(s - m)
//               against the row's running max m, computed before the
//               chunk's own max is known and redone only for a warp in which
//               some row's max grew by more than 2^8 (S is still in tensor
//               memory then); O is rescaled only in that case.  P is written
//               as bf16 over S's columns.  Both tiles' softmaxes run at once.
// Tensor memory (512 columns): S_a | S_b | O_a | O_b.
//
// Two launch shapes:
//  - one split per unit (at least as many units as SMs): each CTA writes
//    O / l straight to the output, and CTAs take the units longest first
//    (every CTA ranks the (sequence, tile pair) groups by chunks x tiles
//    from ctx and N), so the long sequences of a ragged batch start early;
//  - several splits per unit (fewer units than SMs): a cooperative launch,
//    so every CTA is resident at once.  Each split writes its rows' O / l
//    (bf16) and log-sum-exp to the workspace and arrives on its unit's
//    counter; when all splits have arrived, split s combines rows
//    [s R, s R + R) of the unit from L2 and writes them; the last split to
//    leave resets the unit's counters to zero.
// Every wait is bounded (mbarrier waits and the counter spin): on timeout a
// CTA flags LTD_DEVERR_TIMEOUT, drains its own TMA loads and MMAs, still
// arrives and departs on its counter, frees its tensor memory and returns.
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
constexpr int kThreads = 384;  // TMA warp, MMA warp, 2 idle, 8 softmax warps
constexpr int kMaxW32 = LTD_MAX_N / 32;
constexpr int kMaxSplits = 64;
constexpr int kMaxGroups = 1024;  // (sequence, tile pair) groups ranked on the device
constexpr uint32_t kHalf = 16384;      // 128 rows x 128 bytes
constexpr uint32_t kTile = 2 * kHalf;  // 128 x 128 bf16
constexpr uint32_t kOffQ = 0;                                  // Q_a, Q_b
constexpr uint32_t kOffK = kOffQ + 2 * kTile;                  // two stages
constexpr uint32_t kOffV = kOffK + 2 * kTile;                  // two stages
constexpr uint32_t kOffMask = kOffV + 2 * kTile;               // [256][8] words
constexpr uint32_t kOffCost = kOffMask + kRows * kMaxW32 * 4;  // [kMaxGroups] int
constexpr uint32_t kOffOrder = kOffCost + kMaxGroups * 4;      // [kMaxGroups] int
constexpr uint32_t kOffBar = kOffOrder + kMaxGroups * 4;
constexpr uint32_t kOffHolder = kOffBar + 24 * 8;
constexpr uint32_t kSmemBytes = kOffHolder + 16 + 1024;  // + alignment slack
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kRowBytes = kD * 2;     // one bf16 output / partial row
// P may grow to 2^8 before a row's running max is raised: bf16 bits of 2^8
constexpr uint32_t kPMaxBits = 0x4380u;

enum Bar { QFULL = 0, KFULL = 1, VFULL = 3, KEMPTY = 5, VEMPTY = 7, SFULL = 9, PFULL = 11, FIN = 13, CBAR = 14 };

// Optional phase timestamps for performance work (off in normal builds).
#ifdef LTD_TRACE
__device__ unsigned long long g_attn_trace[4096][48];
#define TRACE_VAL(slot, v)                                                                    \
  do {                                                                                        \
    const int cta_ = blockIdx.x + gridDim.x * (blockIdx.y + gridDim.y * blockIdx.z);          \
    if (cta_ < 4096) g_attn_trace[cta_][slot] = (v);                                          \
  } while (0)
#define TRACE(slot) TRACE_VAL(slot, tc::globaltimer())
#else
#define TRACE(slot) \
  do {              \
  } while (0)
#define TRACE_VAL(slot, v) \
  do {                     \
  } while (0)
#endif

struct TcArgs {
  int32_t batch, hq, hkv, G, n_max, s_cap, max_ctx, W32;
  int32_t splits, n_pairs, lpt;
  int32_t nch_h;  // host bound on chunks per sequence: ceil((max_ctx + n_max) / 128)
  int32_t rs;     // rows per combining split: multiple of 4, >= 256 / splits
  const int32_t* ctx;
  const int32_t* n_verify;
  const uint32_t* mask;
  float scale_log2;
  __nv_bfloat16* out;
  uint8_t* part_o;  // [unit][split][256 rows][256 B] O / l, bf16, chunks swizzled (splits > 1)
  float* part_l;    // [unit][split][256] log2-sum-exp
  uint32_t* sync;   // [unit][2] arrive, depart
  const uint8_t* next_k;  // the next call's caches: L2 prefetch targets (or null)
  const uint8_t* next_v;
  uint32_t* err;
  // K and V through one tensor map when both caches fit one 4-D map (the
  // fourth coordinate picks the cache), else one map each
  int32_t kv_one, kv_wk, kv_wv;
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

__device__ __forceinline__ bool seq_ok(const TcArgs& a, int ctx, int N) {
  return N >= 1 && N <= a.n_max && ctx >= 0 && ctx <= a.max_ctx && ctx + N <= a.s_cap;
}

__global__ void __launch_bounds__(kThreads, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tq, const __grid_constant__ CUtensorMap tk,
                   const __grid_constant__ CUtensorMap tv, const TcArgs a) {
  extern __shared__ uint8_t smem_raw[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) TRACE(0);
  const uint32_t raw = tc::smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  uint32_t* mask_s = reinterpret_cast<uint32_t*>(gbase + kOffMask);
  uint32_t* holder = reinterpret_cast<uint32_t*>(gbase + kOffHolder);
  auto bar = [&](int i) { return base + kOffBar + 8u * i; };
  const int S = a.splits;

  if (tid == 0) {
    tc::tma_prefetch(&tq);
    tc::tma_prefetch(&tk);
    if (!a.kv_one) tc::tma_prefetch(&tv);
    TRACE(42);
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
    tc::mbar_init(bar(CBAR), 1);
    tc::mbar_init_fence();
    TRACE(19);
  }
  // everything above touches only shared memory and this launch's
  // parameters; what follows may read another kernel's output
  grid_wait();
  trigger_dependents();
  if (tid == 0) TRACE(43);

  // ------------------------------------------------------ which unit
  int split = 0, pair, b, kvh;
  if (S > 1) {
    split = blockIdx.x;
    pair = blockIdx.y;
    b = blockIdx.z / a.hkv;
    kvh = blockIdx.z % a.hkv;
  } else {
    const int i = blockIdx.x;
    int g = i / a.hkv;
    kvh = i % a.hkv;
    if (a.lpt) {
      // rank every (sequence, tile pair) group by its work, largest first
      // (ties to the lower group, so equal pairs of one sequence, which
      // read the same K/V, stay together), and take the group at this
      // CTA's rank; bad sequences rank last and flag on their own CTAs
      int* cost = reinterpret_cast<int*>(gbase + kOffCost);
      int* order = reinterpret_cast<int*>(gbase + kOffOrder);
      const int groups = a.batch * a.n_pairs;
      for (int gi = tid; gi < groups; gi += kThreads) {
        const int bb = gi / a.n_pairs, pp = gi % a.n_pairs;
        const int c = a.ctx[bb], n = a.n_verify[bb];
        int w = 0;
        if (seq_ok(a, c, n)) {
          const int rows = n * a.G - pp * kRows;
          w = (rows <= 0 ? 0 : (rows > kBM ? 2 : 1)) * ((c + n + kBN - 1) / kBN);
        }
        cost[gi] = w;
      }
      __syncthreads();
      for (int gi = tid; gi < groups; gi += kThreads) {
        const int w = cost[gi];
        int r = 0;
        for (int o = 0; o < groups; ++o) {
          const int wo = cost[o];
          r += (wo > w) || (wo == w && o < gi);
        }
        order[r] = gi;
      }
      __syncthreads();
      g = order[g];
    }
    b = g / a.n_pairs;
    pair = g % a.n_pairs;
  }
  if (tid == 0) TRACE_VAL(25, static_cast<unsigned long long>(clock64()));
  if (tid == 0) TRACE(26);

  // Keys are split by the host bound on the chunk count, so a split knows
  // its first chunk before reading ctx and N: the loads of Q and of the
  // first K chunk go out at once (extra ones past this sequence's end are
  // drained and ignored).  V of that chunk and the later chunks wait for the
  // producer loop after the setup, so no CTA's first S queues at the DRAM
  // behind every CTA's other chunks (8B-class layer 15.8 -> 15.1 us,
  // 13B-class 20.1 -> 18.9 us).
  const int cs = split * a.nch_h / S, ce = (split + 1) * a.nch_h / S;
  const int kvrow = b * a.hkv + kvh;
  const int row0 = pair * kRows;
  const bool has_b_h = row0 + kBM < a.n_max * a.G;  // tile b may hold rows
  int nk_issued[2] = {0, 0}, nv_issued[2] = {0, 0}, n_issued = 0;
  bool q_issued = false, v0_owed = false;
  auto issue_k = [&](int j) {
    const int st = j & 1;
    tc::mbar_expect_tx(bar(KFULL + st), kTile);
    for (int h = 0; h < 2; ++h)
      tc::tma_load_4d(base + kOffK + st * kTile + h * kHalf, &tk, bar(KFULL + st), h * 64,
                      (cs + j) * kBN, kvrow, a.kv_wk);
    ++nk_issued[st];
  };
  auto issue_v = [&](int j) {
    const int st = j & 1;
    tc::mbar_expect_tx(bar(VFULL + st), kTile);
    for (int h = 0; h < 2; ++h)
      tc::tma_load_4d(base + kOffV + st * kTile + h * kHalf, a.kv_one ? &tk : &tv, bar(VFULL + st),
                      h * 64, (cs + j) * kBN, kvrow, a.kv_wv);
    ++nv_issued[st];
  };
  auto issue_first = [&]() {
    tc::mbar_expect_tx(bar(QFULL), has_b_h ? 2 * kTile : kTile);
    for (int t = 0; t < (has_b_h ? 2 : 1); ++t) {
      const int qrow = b * a.n_max + (row0 + t * kBM) / a.G;
      for (int h = 0; h < 2; ++h)
        tc::tma_load_3d(base + kOffQ + t * kTile + h * kHalf, &tq, bar(QFULL), h * 64, kvh * a.G,
                        qrow);
    }
    q_issued = true;
    TRACE(20);
    if (ce - cs > 0) {
      issue_k(0);
      TRACE(44);
      v0_owed = true;
    }
    TRACE(17);
  };
  // every load a CTA issued lands before it leaves or reuses shared memory
  auto drain = [&]() {
    if (q_issued) tc::mbar_wait(bar(QFULL), 0);
    for (int st = 0; st < 2; ++st) {
      if (nk_issued[st] > 0) tc::mbar_wait(bar(KFULL + st), (nk_issued[st] - 1) & 1);
      if (nv_issued[st] > 0) tc::mbar_wait(bar(VFULL + st), (nv_issued[st] - 1) & 1);
    }
  };
  if (tid == 0 && !a.lpt) issue_first();

  // Everything a CTA returns early on is shared by all splits of its unit.
  const int ctx = a.ctx[b];
  const int N = a.n_verify[b];
  const int M = N * a.G;
  if (tid == 0) TRACE(21);
  if (!seq_ok(a, ctx, N) || row0 >= M) {
    if (tid == 0) {
      if (!seq_ok(a, ctx, N) && split == 0 && pair == 0 && kvh == 0)
        flag_error(a.err, (N < 1 || N > a.n_max) ? LTD_DEVERR_NVERIFY : LTD_DEVERR_CTX);
      drain();
    }
    return;
  }
  const bool has_b = row0 + kBM < M;
  const int nk = ctx + N;
  const int nch = (nk + kBN - 1) / kBN;
  const int nc = max(0, min(ce, nch) - cs);
  const int key_lo = cs * kBN, key_hi = min(ce * kBN, nk);

  if (tid == 0 && a.lpt) issue_first();
  if (warp == 1) {
    tc::tmem_alloc(tc::smem_u32(holder), kTmemCols);
    tc::tmem_relinquish();
  }
  // softmax threads (warps 4-11): tile x, TMEM lane lrow, row rr of the unit
  const bool smx = warp >= 4;
  const int x = (warp - 4) >> 2;
  const int lrow = 32 * (warp & 3) + lane;
  const int rr = kBM * x + lrow;
  const int R = row0 + rr;
  const bool row_ok = smx && R < M;
  if (smx) {
    const int slot = R / a.G;
    const bool in = slot < a.n_max;
    for (int w = 0; w < a.W32; ++w)
      mask_s[rr * kMaxW32 + w] =
          in ? a.mask[(static_cast<int64_t>(b) * a.n_max + slot) * a.W32 + w] : 0u;
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = holder[0];
  if (tid == 0) TRACE(1);
  bool ok = true;
  const bool tile_active = smx && (x == 0 || has_b) && nc > 0;
  float m = -CUDART_INF_F, l = 0.f;  // the row's running max (log2 units) and sum

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
#ifdef LTD_TRACE
      unsigned long long w_empty = 0, t_e = 0;
#endif
      if (v0_owed) {
        issue_v(0);
        n_issued = 1;
      }
      for (int j = n_issued; j < nc && ok; ++j) {
        const int st = j & 1;
#ifdef LTD_TRACE
        t_e = tc::globaltimer();
#endif
        ok = tc::mbar_wait(bar(KEMPTY + st), ((j >> 1) - 1) & 1);
        if (!ok) break;
        issue_k(j);
        ok = tc::mbar_wait(bar(VEMPTY + st), ((j >> 1) - 1) & 1);
        if (!ok) break;
        issue_v(j);
#ifdef LTD_TRACE
        w_empty += tc::globaltimer() - t_e;
#endif
      }
      TRACE_VAL(32, w_empty);
      drain();
      if (!ok) flag_error(a.err, LTD_DEVERR_TIMEOUT);
      if (a.next_k != nullptr && nc > 0) {
        // this CTA's loads have landed: ask L2 for the same rows of the next
        // call's caches, 128 rows (32 KB) per request
        const int r_end = min(key_hi, key_lo + nc * kBN);
        for (int r = key_lo; r < r_end; r += kBN) {
          const uint32_t bytes = static_cast<uint32_t>(min(kBN, r_end - r)) * kRowBytes;
          const int64_t off = (static_cast<int64_t>(kvrow) * a.s_cap + r) * kRowBytes;
          tc::prefetch_l2(a.next_k + off, bytes);
          tc::prefetch_l2(a.next_v + off, bytes);
        }
      }
    }
  } else if (warp == 1) {
    // ----------------------------------------------------------------- MMA
    if (lane == 0 && nc > 0) {
      const uint32_t id_s = tc::idesc_bf16(kBM, kBN, false);
      const uint32_t id_o = tc::idesc_bf16(kBM, kD, true);
      const int ntile = has_b ? 2 : 1;
      // Every shared-memory descriptor is computed once, so the issue loop
      // below is MMA instructions only (the thread shares its scheduler with
      // two softmax warps, and each MMA lasts just 64 cycles).
      uint64_t dq[2][8], dk[2][8], dv[2][8];
#pragma unroll
      for (int u = 0; u < 2; ++u) {
#pragma unroll
        for (int ks = 0; ks < 8; ++ks) {
          dq[u][ks] = tc::sdesc_sw128(base + kOffQ + u * kTile + (ks >> 2) * kHalf + (ks & 3) * 32, 16, 1024);
          dk[u][ks] = tc::sdesc_sw128(base + kOffK + u * kTile + (ks >> 2) * kHalf + (ks & 3) * 32, 16, 1024);
          dv[u][ks] = tc::sdesc_sw128(base + kOffV + u * kTile + ks * 2048, kHalf, 1024);
        }
      }
      // (t and st are compile-time constants at every call)
      auto issue_s = [&](int t, int st) {
#pragma unroll
        for (int ks = 0; ks < 8; ++ks)
          tc::mma_bf16(tmem + t * kBN, dq[t][ks], dk[st][ks], id_s, ks > 0 ? 1u : 0u);
      };
      auto issue_pv = [&](int t, int st, uint32_t acc) {
#pragma unroll
        for (int ks = 0; ks < 8; ++ks)
          tc::mma_bf16_ts(tmem + 2 * kBN + t * kD, tmem + t * kBN + 8 * ks, dv[st][ks], id_o,
                          ks > 0 ? 1u : acc);
      };
#ifdef LTD_TRACE
      unsigned long long w_load = 0, w_p = 0, t_w;
#define TW_BEGIN() t_w = tc::globaltimer()
#define TW_END(acc) acc += tc::globaltimer() - t_w
#else
#define TW_BEGIN() \
  do {             \
  } while (0)
#define TW_END(acc) \
  do {              \
  } while (0)
#endif
      ok = tc::mbar_wait(bar(QFULL), 0);
      TRACE(2);
      if (ok) ok = tc::mbar_wait(bar(KFULL + 0), 0);
      TRACE(3);
      if (ok) {
        tc::fence_after_sync();
        issue_s(0, 0);
        tc::mma_commit(bar(SFULL + 0));
        if (ntile > 1) {
          issue_s(1, 0);
          tc::mma_commit(bar(SFULL + 1));
        }
        tc::mma_commit(bar(KEMPTY + 0));
      }
      // chunk j in stage st = j & 1: PV_x(j) and S_x(j+1) per tile
      auto step = [&](int j, int st) -> bool {
        const bool nxt = j + 1 < nc;
        TW_BEGIN();
        bool k = tc::mbar_wait(bar(VFULL + st), (j >> 1) & 1);
        if (k && nxt) k = tc::mbar_wait(bar(KFULL + (st ^ 1)), ((j + 1) >> 1) & 1);
        TW_END(w_load);
        const uint32_t acc = j > 0 ? 1u : 0u;
#pragma unroll
        for (int t = 0; t < 2; ++t) {
          if (!k || t >= ntile) break;
          TW_BEGIN();
          k = tc::mbar_wait(bar(PFULL + t), j & 1);
          TW_END(w_p);
          if (!k) break;
          tc::fence_after_sync();
          issue_pv(t, st, acc);
          if (nxt) {
            issue_s(t, st ^ 1);
            tc::mma_commit(bar(SFULL + t));
          }
        }
        if (!k) return false;
        if (nxt) tc::mma_commit(bar(KEMPTY + (st ^ 1)));
        tc::mma_commit(bar(VEMPTY + st));
        return true;
      };
      for (int j = 0; j < nc && ok; j += 2) {
        ok = step(j, 0);
        if (ok && j + 1 < nc) ok = step(j + 1, 1);
      }
      TRACE_VAL(22, w_load);
      TRACE_VAL(24, w_p);
      TRACE_VAL(29, static_cast<unsigned long long>(nc));
      TRACE(31);
#undef TW_BEGIN
#undef TW_END
      // every MMA of this CTA completes before tensor memory is read or freed
      tc::mma_commit(bar(FIN));
      tc::mbar_wait(bar(FIN), 0);
      if (!ok) flag_error(a.err, LTD_DEVERR_TIMEOUT);
    }
  } else if (tile_active) {
    // ------------------------------------------------------------- softmax
    const uint32_t lane_off = (32u * (warp & 3)) << 16;
    const uint32_t t_s = tmem + x * kBN + lane_off;
    const uint32_t t_o = tmem + 2 * kBN + x * kD + lane_off;
    const uint32_t* mbits = mask_s + rr * kMaxW32;
    const int vis_all_below = min(ctx, key_hi);  // keys below this are all visible
    const float sl2 = a.scale_log2;
    const int w32 = a.W32;
    const bool tr = (tid & 127) == 0;
#ifdef LTD_TRACE
    unsigned long long w_s = 0, t_s0 = 0;
#endif
    for (int j = 0; j < nc; ++j) {
#ifdef LTD_TRACE
      t_s0 = tc::globaltimer();
#endif
      ok = tc::mbar_wait(bar(SFULL + x), j & 1);
#ifdef LTD_TRACE
      w_s += tc::globaltimer() - t_s0;
#endif
      ok = __all_sync(0xFFFFFFFFu, ok);
      if (tr && j < 2) TRACE(4 + 4 * x + 2 * j);
      if (!ok) break;
      tc::fence_after_sync();
      const int kbase = key_lo + j * kBN;
      const bool all_vis = row_ok && kbase + kBN <= vis_all_below;
      // P against the row's running max m (a row without one yet first takes
      // this chunk's max); the chunk's own max is tracked on the way and, if
      // it exceeds the reference by more than 2^8 in some row of the warp,
      // the warp re-derives P from S, still intact in tensor memory, 32
      // columns at a time.
      tc::Frag128 f;
      float mref = m;
      float2 ls2 = make_float2(0.f, 0.f);
      uint32_t vq[4] = {0xFFFFFFFFu, 0xFFFFFFFFu, 0xFFFFFFFFu, 0xFFFFFFFFu};
      if (!all_vis) {
#pragma unroll
        for (int qq = 0; qq < 4; ++qq)
          vq[qq] = row_ok ? visible32(kbase + 32 * qq, ctx, key_hi, w32, mbits) : 0u;
      }
      __syncwarp();  // the load below is warp-collective; the branch above is per row
      tc::tmem_ld128_sync(t_s, f);
      if (tr && j == 0 && x == 0) TRACE(27);
      if (!all_vis) {
#pragma unroll
        for (int c = 0; c < 128; ++c)
          f.r[c] = ((vq[c >> 5] >> (c & 31)) & 1u) ? f.r[c] : 0xFF800000u;  // -inf if hidden
      }
      if (__any_sync(0xFFFFFFFFu, mref == -CUDART_INF_F)) {
        float r8[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) r8[u] = __uint_as_float(f.r[u]);
#pragma unroll
        for (int c = 8; c < 128; c += 16) {
#pragma unroll
          for (int u = 0; u < 8; ++u)
            r8[u] = tc::fmax3(r8[u], __uint_as_float(f.r[c + 2 * u]), __uint_as_float(f.r[c + 2 * u + 1]));
        }
        const float cm = fmaxf(tc::fmax3(r8[0], r8[1], r8[2]),
                               fmaxf(tc::fmax3(r8[3], r8[4], r8[5]), fmaxf(r8[6], r8[7]))) * sl2;
        if (mref == -CUDART_INF_F) mref = cm;
      }
      // bf16 of P >= 0 orders like an unsigned integer, so the largest P
      // is the largest 16-bit half of the packed registers
      uint32_t pmax2 = 0u;
      {
        const float mz = (mref == -CUDART_INF_F) ? 0.f : mref;  // -inf only if all are hidden
        const float2 sl22 = make_float2(sl2, sl2), nm2 = make_float2(-mz, -mz);
        // P packed in place: pair c is read from registers 2c, 2c+1 and
        // written to register c (c <= 2c, so nothing unread is overwritten)
#pragma unroll
        for (int c = 0; c < 64; ++c) {
          const float2 t = __ffma2_rn(
              make_float2(__uint_as_float(f.r[2 * c]), __uint_as_float(f.r[2 * c + 1])), sl22, nm2);
          const float2 pp = make_float2(tc::ex2(t.x), tc::ex2(t.y));
          ls2 = __fadd2_rn(ls2, pp);
          f.r[c] = pack_bf16(pp.x, pp.y);
          pmax2 = __vmaxu2(pmax2, f.r[c]);
        }
      }
      // P above 2^8 means the chunk max passed m + 8
      const bool over = max(pmax2 & 0xFFFFu, pmax2 >> 16) > kPMaxBits;
      if (!__any_sync(0xFFFFFFFFu, over)) {
        tc::tmem_st64_lo_sync(t_s, f);
      } else {
        // S is still intact in tensor memory: take the chunk's max, then
        // derive P again, 32 columns at a time (P columns 16 qq .. 16 qq + 15
        // overlie S columns already read)
        float cm = -CUDART_INF_F;
#pragma unroll 1
        for (int qq = 0; qq < 4; ++qq) {
          tc::Frag32 g;
          tc::tmem_ld32_sync(t_s + 32 * qq, g);
          const uint32_t v = qq == 0 ? vq[0] : (qq == 1 ? vq[1] : (qq == 2 ? vq[2] : vq[3]));
#pragma unroll
          for (int c = 0; c < 32; ++c)
            if ((v >> c) & 1u) cm = fmaxf(cm, __uint_as_float(g.r[c]));
        }
        if (over) mref = cm * sl2;
        const float mz = (mref == -CUDART_INF_F) ? 0.f : mref;
        const float2 sl22 = make_float2(sl2, sl2), nm2 = make_float2(-mz, -mz);
        ls2 = make_float2(0.f, 0.f);
#pragma unroll 1
        for (int qq = 0; qq < 4; ++qq) {
          tc::Frag32 g;
          tc::tmem_ld32_sync(t_s + 32 * qq, g);
          const uint32_t v = qq == 0 ? vq[0] : (qq == 1 ? vq[1] : (qq == 2 ? vq[2] : vq[3]));
          tc::Frag16 pf;
#pragma unroll
          for (int c = 0; c < 16; ++c) {
            const float s0 = ((v >> (2 * c)) & 1u) ? __uint_as_float(g.r[2 * c]) : -CUDART_INF_F;
            const float s1 = ((v >> (2 * c + 1)) & 1u) ? __uint_as_float(g.r[2 * c + 1]) : -CUDART_INF_F;
            const float2 t = __ffma2_rn(make_float2(s0, s1), sl22, nm2);
            const float2 pp = make_float2(tc::ex2(t.x), tc::ex2(t.y));
            ls2 = __fadd2_rn(ls2, pp);
            pf.r[c] = pack_bf16(pp.x, pp.y);
          }
          tc::tmem_st16_sync(t_s + 16 * qq, pf);
        }
      }
      if (tr && j == 0 && x == 0) TRACE(28);
      // S(j) complete implies P_x(j-1) V finished, so O_x is stable here
      const bool need = (mref != m) && (m != -CUDART_INF_F);
      const float alpha = need ? tc::ex2(m - mref) : 1.f;
      if (__any_sync(0xFFFFFFFFu, need)) {
#pragma unroll 1
        for (int qq = 0; qq < 4; ++qq) {
          tc::Frag32 o;
          tc::tmem_ld32_sync(t_o + 32 * qq, o);
#pragma unroll
          for (int c = 0; c < 32; ++c) o.r[c] = __float_as_uint(__uint_as_float(o.r[c]) * alpha);
          tc::tmem_st32_sync(t_o + 32 * qq, o);
        }
      }
      m = mref;
      l = l * alpha + (ls2.x + ls2.y);
      if (x == 0 && kbase + kBN > key_hi) {
        // Keys from key_hi on may hold anything in the cache, even NaN: P is
        // 0 there, but 0 * NaN is not, so tile a's threads clear those V rows
        // (both 64-dim halves) before either tile's PV reads this stage.
        const int st = j & 1;
        // (a failed wait is flagged; the MMA thread times out on the same stage)
        if (!__all_sync(0xFFFFFFFFu, tc::mbar_wait(bar(VFULL + st), (j >> 1) & 1)) && lane == 0)
          flag_error(a.err, LTD_DEVERR_TIMEOUT);
        const int z0 = key_hi - kbase;  // 1 .. 127
        uint4* vs = reinterpret_cast<uint4*>(gbase + kOffV + st * kTile);
        for (int idx = lrow; idx < (kBN - z0) * 16; idx += kBM) {
          const int row = z0 + (idx >> 4), piece = idx & 15;
          vs[((piece >> 3) * kHalf + row * 128) / 16 + (piece & 7)] = make_uint4(0u, 0u, 0u, 0u);
        }
        tc::fence_smem_async();
      }
      __syncwarp();  // the zeroing loop above runs per thread; the wait is warp-collective
      tc::tmem_wait_st();
      if (tr && j == 0 && x == 0) TRACE(30);
      tc::fence_before_sync();
      tc::mbar_arrive(bar(PFULL + x));
      if (tr && j < 2) TRACE(5 + 4 * x + 2 * j);
    }
    if (ok) {
      ok = tc::mbar_wait(bar(FIN), 0);
      ok = __all_sync(0xFFFFFFFFu, ok);
    }
    if (tr) TRACE(12 + x);
    if (tr) TRACE_VAL(33 + x, w_s);
    if (!ok && lane == 0) flag_error(a.err, LTD_DEVERR_TIMEOUT);
  }

  // --------------------------------------------------------- epilogue
  // O / l of every row (bf16; zero where a row has nothing) and its
  // log2-sum-exp are staged in shared memory over Q and over the mask (both
  // free once the last MMA has completed): row r's 16-byte chunk c sits at
  // ((c ^ (r & 15)) << 4), so the row-per-thread stores of a warp spread
  // over the banks.  One split: all threads copy the rows to the output,
  // coalesced.  Several: the partial layout below.
  const int unit = (b * a.hkv + kvh) * a.n_pairs + pair;
  const int Mv = min(kRows, M - row0);
  // the producer has drained every load (Q included) and the MMAs are done
  // before the staging below overwrites Q
  tc::fence_before_sync();
  __syncthreads();
  uint8_t* stg = gbase + kOffQ;
  float* stg_l = reinterpret_cast<float*>(gbase + kOffMask);
  // tcgen05.ld is warp-collective: the O load is taken by whole warps
  // (tile_active and ok are uniform within a warp), the writes per row.
  const bool loaded = tile_active && ok;
  tc::Frag128 o;
  if (loaded) {
    tc::fence_after_sync();
    tc::tmem_ld128_sync(tmem + 2 * kBN + x * kD + ((32u * (warp & 3)) << 16), o);
  }
  if (row_ok) {
    const bool have = loaded && l > 0.f;
    const float inv = have ? 1.f / l : 0.f;
    uint8_t* srow = stg + rr * kRowBytes;
#pragma unroll
    for (int c = 0; c < 16; ++c) {
      uint4 w = make_uint4(0u, 0u, 0u, 0u);
      if (have) {
        w.x = pack_bf16(__uint_as_float(o.r[8 * c]) * inv, __uint_as_float(o.r[8 * c + 1]) * inv);
        w.y = pack_bf16(__uint_as_float(o.r[8 * c + 2]) * inv, __uint_as_float(o.r[8 * c + 3]) * inv);
        w.z = pack_bf16(__uint_as_float(o.r[8 * c + 4]) * inv, __uint_as_float(o.r[8 * c + 5]) * inv);
        w.w = pack_bf16(__uint_as_float(o.r[8 * c + 6]) * inv, __uint_as_float(o.r[8 * c + 7]) * inv);
      }
      *reinterpret_cast<uint4*>(srow + ((c ^ (rr & 15)) << 4)) = w;
    }
    stg_l[rr] = have ? m + __log2f(l) : -CUDART_INF_F;
  }
  tc::fence_smem_async();  // the staging is read by bulk copies
  tc::fence_before_sync();
  __syncthreads();
  if (tid == 0) TRACE(14);
  if (warp == 1) {
    __syncwarp();
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, kTmemCols);
  }
  if (S == 1) {
    for (int idx = tid; idx < Mv * 16; idx += kThreads) {
      const int r = idx >> 4, c = idx & 15;
      const int Rr = row0 + r, slot = Rr / a.G, g = Rr % a.G;
      const uint4 v = *reinterpret_cast<const uint4*>(stg + r * kRowBytes + ((c ^ (r & 15)) << 4));
      reinterpret_cast<uint4*>(a.out + ((static_cast<int64_t>(b) * a.n_max + slot) * a.hq +
                                        kvh * a.G + g) * kD)[c] = v;
    }
    return;
  }

  // ------------------------------------- combine the splits (S > 1 only)
  // Each split stores its staged rows and sums with one bulk copy each
  // (split-major: [unit][split][row]); rows [o rs, o rs + rs) of a unit are
  // combined by its split o ("owner"), which pulls that block of every
  // split with one bulk copy per split.
  const int Rs = a.rs;
  uint32_t* arrive = a.sync + 2 * unit;
  uint32_t* depart = arrive + 1;
  if (tid == 0) {
    const int64_t pb = static_cast<int64_t>(unit) * S + split;
    tc::bulk_s2g(a.part_o + pb * kRows * kRowBytes, base + kOffQ, Mv * kRowBytes);
    tc::bulk_s2g(a.part_l + pb * kRows, base + kOffMask, ((Mv + 3) & ~3) * 4);
    tc::bulk_commit();
    tc::bulk_wait_all();
    tc::fence_proxy_async_global();
    tc::red_add_release_gpu(arrive, 1u);
    bool got = tc::ld_acquire_gpu(arrive) >= static_cast<uint32_t>(S);
    if (!got) {
      const uint64_t t0 = tc::globaltimer();
      while (!got) {
        __nanosleep(32);
        got = tc::ld_acquire_gpu(arrive) >= static_cast<uint32_t>(S);
        if (!got && tc::globaltimer() - t0 > tc::kWaitLimitNs) break;
      }
    }
    if (!got) flag_error(a.err, LTD_DEVERR_TIMEOUT);
    holder[1] = got ? 1u : 0u;
    TRACE(15);
  }
  __syncthreads();
  const int r_lo = split * Rs;
  const int nrows = max(0, min(Mv, r_lo + Rs) - r_lo);
  if (holder[1] != 0u && nrows > 0) {
    if (tid == 0) {
      // the acquire above orders the other splits' stores before these reads
      tc::fence_proxy_async_global();
      const int nl = min(Rs, kRows - r_lo);  // a multiple of 4
      tc::mbar_expect_tx(bar(CBAR), static_cast<uint32_t>(S) * (nrows * kRowBytes + nl * 4));
      for (int p = 0; p < S; ++p) {
        const int64_t pb = static_cast<int64_t>(unit) * S + p;
        tc::bulk_g2s(base + kOffK + p * Rs * kRowBytes, a.part_o + (pb * kRows + r_lo) * kRowBytes,
                     nrows * kRowBytes, bar(CBAR));
        tc::bulk_g2s(base + kOffMask + p * Rs * 4, a.part_l + pb * kRows + r_lo, nl * 4, bar(CBAR));
      }
    }
    // CTA-uniform, as a barrier follows under it
    const bool in = __syncthreads_and(tc::mbar_wait(bar(CBAR), 0)) != 0;
    if (tid == 0) TRACE(18);
    if (!in) {
      if (tid == 0) flag_error(a.err, LTD_DEVERR_TIMEOUT);
    } else {
      const uint8_t* cin = gbase + kOffK;
      const float* lin = reinterpret_cast<const float*>(gbase + kOffMask);
      // A thread per (row, 16-byte chunk): the splits' log2-sum-exps give
      // the row's max, then each split's weight 2^(lse_p - max) and its chunk
      // are fetched with independent shared loads (four splits in flight)
      // and accumulated; every split wrote every row below Mv (zeros where
      // it had no keys).
      for (int idx = tid; idx < nrows * 16; idx += kThreads) {
        const int r = idx >> 4, c = idx & 15;
        const float* lr = lin + r;
        float mx = -CUDART_INF_F;
#pragma unroll 4
        for (int p = 0; p < S; ++p) mx = fmaxf(mx, lr[p * Rs]);
        float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        float L = 0.f;
        if (mx > -CUDART_INF_F) {
          // rows keep the staging's chunk swizzle (by row within the unit)
          const uint8_t* cr = cin + r * kRowBytes + ((c ^ ((r_lo + r) & 15)) << 4);
#pragma unroll 4
          for (int p = 0; p < S; ++p) {
            const float w = tc::ex2(lr[p * Rs] - mx);  // 0 for a split without keys
            const uint4 v = *reinterpret_cast<const uint4*>(cr + p * Rs * kRowBytes);
            L += w;
            const uint32_t e[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
            for (int t = 0; t < 4; ++t) {
              acc[2 * t] = fmaf(w, __uint_as_float(e[t] << 16), acc[2 * t]);
              acc[2 * t + 1] = fmaf(w, __uint_as_float(e[t] & 0xFFFF0000u), acc[2 * t + 1]);
            }
          }
        }
        const float inv = L > 0.f ? 1.f / L : 0.f;
        const int Rr = row0 + r_lo + r;
        const int slot = Rr / a.G, g = Rr % a.G;
        uint4 w;
        w.x = pack_bf16(acc[0] * inv, acc[1] * inv);
        w.y = pack_bf16(acc[2] * inv, acc[3] * inv);
        w.z = pack_bf16(acc[4] * inv, acc[5] * inv);
        w.w = pack_bf16(acc[6] * inv, acc[7] * inv);
        reinterpret_cast<uint4*>(a.out + ((static_cast<int64_t>(b) * a.n_max + slot) * a.hq +
                                          kvh * a.G + g) * kD)[c] = w;
      }
      if (tid == 0) TRACE(23);
    }
  }
  __syncthreads();
  if (tid == 0) {
    TRACE(16);
    // every split of this unit has passed its spin once all have departed
    const uint32_t d = atomicAdd(depart, 1u);
    if (d == static_cast<uint32_t>(S) - 1u) {
      atomicExch(arrive, 0u);
      atomicExch(depart, 0u);
    }
  }
}

struct Plan {
  int n_pairs, splits, units, lpt, nch, rs;
};

// Streaming multiprocessors of the current device (152 if it cannot be asked).
int device_sms() {
  static std::mutex mu;
  static int known[128] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 128) {
    (void)cudaGetLastError();
    return 152;
  }
  std::lock_guard<std::mutex> lock(mu);
  if (known[dev] == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1) {
      (void)cudaGetLastError();
      n = 152;
    }
    known[dev] = n;
  }
  return known[dev];
}

// Units = (sequence, KV head, tile pair).  With fewer units than SMs each
// unit's keys are cut into the fewest splits that give the shortest longest
// split, at most SMs / units of them, so all CTAs fit one wave.
Plan plan(int32_t batch, int32_t hq, int32_t hkv, int32_t n_max, int32_t max_ctx) {
  const int G = hq / hkv;
  Plan p{};
  p.n_pairs = (n_max * G + kRows - 1) / kRows;
  const int64_t units = static_cast<int64_t>(batch) * hkv * p.n_pairs;
  p.units = static_cast<int>(units);
  const int nch = (max_ctx + n_max + kBN - 1) / kBN;
  const int sms = device_sms();
  p.splits = 1;
  if (units < sms) {
    int smax = static_cast<int>(sms / units);
    smax = smax < nch ? smax : nch;
    smax = smax < kMaxSplits ? smax : kMaxSplits;
    if (smax > 1) {
      const int maxc = (nch + smax - 1) / smax;
      p.splits = (nch + maxc - 1) / maxc;
    }
  }
  p.lpt = (p.splits == 1 && static_cast<int64_t>(batch) * p.n_pairs <= kMaxGroups) ? 1 : 0;
  p.nch = nch;
  p.rs = (((kRows + p.splits - 1) / p.splits) + 3) & ~3;
  return p;
}

size_t align256(size_t n) { return (n + 255) / 256 * 256; }

struct WsLayout {
  size_t part_o, part_l, sync, total;
};
WsLayout ws_layout(const Plan& pl) {
  WsLayout w{};
  if (pl.splits <= 1) return w;
  // [unit][split][256] rows
  const size_t rows = static_cast<size_t>(pl.units) * pl.splits * kRows;
  w.part_o = 0;
  w.part_l = align256(rows * kRowBytes);
  w.sync = w.part_l + align256(rows * sizeof(float));
  w.total = w.sync + align256(static_cast<size_t>(pl.units) * 2 * sizeof(uint32_t));
  return w;
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

namespace {
bool encode_tmap_bf16_4d(CUtensorMap* map, const void* base, uint64_t d0, uint64_t d1, uint64_t d2,
                         uint64_t d3, uint64_t stride1, uint64_t stride2, uint64_t stride3, uint32_t b0,
                         uint32_t b1, uint32_t b2, uint32_t b3) {
  EncodeFn fn = encode_fn();
  if (fn == nullptr) return false;
  const cuuint64_t dims[4] = {d0, d1, d2, d3};
  const cuuint64_t strides[3] = {stride1, stride2, stride3};
  const cuuint32_t box[4] = {b0, b1, b2, b3};
  const cuuint32_t estr[4] = {1, 1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}
}  // namespace

bool attn_tc_supported(const AttnParams& p, ltd_dtype dtype) {
  if (dtype != LTD_BF16 || p.d != kD || p.hkv < 1 || p.hq % p.hkv != 0) return false;
  const int G = p.hq / p.hkv;
  return G >= 1 && G <= kBM && kBM % G == 0 && p.n_max <= LTD_MAX_N;
}


size_t attn_tc_workspace(int32_t batch, int32_t hq, int32_t hkv, int32_t, int32_t n_max,
                         int32_t max_ctx) {
  return ws_layout(plan(batch, hq, hkv, n_max, max_ctx)).total;
}

int32_t attn_tc_launches(int32_t, int32_t, int32_t, int32_t, int32_t) { return 1; }

cudaError_t launch_attn_tc(const AttnParams& p, cudaStream_t s) {
  const Plan pl = plan(p.batch, p.hq, p.hkv, p.n_max, p.max_ctx);
  const WsLayout wl = ws_layout(pl);
  if (p.ws_bytes < wl.total || (wl.total > 0 && p.ws == nullptr)) return cudaErrorInvalidValue;
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
  a.lpt = pl.lpt;
  a.nch_h = pl.nch;
  a.rs = pl.rs;
  a.ctx = p.ctx;
  a.n_verify = p.n_verify;
  a.mask = p.mask;
  a.scale_log2 = p.scale * 1.4426950408889634f;
  a.out = static_cast<__nv_bfloat16*>(p.out);
  uint8_t* ws = static_cast<uint8_t*>(p.ws);
  a.part_o = pl.splits > 1 ? ws + wl.part_o : nullptr;
  a.part_l = pl.splits > 1 ? reinterpret_cast<float*>(ws + wl.part_l) : nullptr;
  a.sync = pl.splits > 1 ? reinterpret_cast<uint32_t*>(ws + wl.sync) : nullptr;
  a.err = p.err;
  // the hint only while one layer's keys and values fit well inside L2
  const uint64_t layer_kv = static_cast<uint64_t>(p.batch) * p.hkv *
                            (static_cast<uint64_t>(p.max_ctx) + p.n_max) * kRowBytes * 2;
  if (p.next_k != nullptr && p.next_v != nullptr && layer_kv <= (64ull << 20)) {
    a.next_k = static_cast<const uint8_t*>(p.next_k);
    a.next_v = static_cast<const uint8_t*>(p.next_v);
  }

  CUtensorMap tq, tk, tv;
  const uint64_t row = kD * 2;
  if (!encode_tmap_bf16_3d(&tq, p.q, kD, p.hq, static_cast<uint64_t>(p.batch) * p.n_max, row,
                           row * p.hq, 64, a.G, kBM / a.G))
    return cudaErrorInvalidValue;
  // One map for both caches saves the kernel a descriptor fetch, which a
  // launch otherwise waits for behind its own first loads.
  const uint64_t rows_kv = static_cast<uint64_t>(p.batch) * p.hkv;
  const uint64_t ka = reinterpret_cast<uint64_t>(p.k), va = reinterpret_cast<uint64_t>(p.v);
  const uint64_t lo = ka < va ? ka : va, gap = ka < va ? va - ka : ka - va;
  a.kv_one = gap > 0 && gap % 16 == 0 && gap < (1ull << 40) &&
             encode_tmap_bf16_4d(&tk, reinterpret_cast<const void*>(lo), kD, p.s_cap, rows_kv, 2, row,
                                 row * p.s_cap, gap, 64, kBN, 1, 1);
  if (a.kv_one) {
    a.kv_wk = ka < va ? 0 : 1;
    a.kv_wv = 1 - a.kv_wk;
    tv = tk;
  } else {
    const uint64_t whole = row * p.s_cap * rows_kv;
    a.kv_wk = a.kv_wv = 0;
    if (!encode_tmap_bf16_4d(&tk, p.k, kD, p.s_cap, rows_kv, 1, row, row * p.s_cap, whole, 64, kBN, 1, 1) ||
        !encode_tmap_bf16_4d(&tv, p.v, kD, p.s_cap, rows_kv, 1, row, row * p.s_cap, whole, 64, kBN, 1, 1))
      return cudaErrorInvalidValue;
  }
  cudaError_t e = cudaFuncSetAttribute(attn_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(kSmemBytes));
  if (e != cudaSuccess) return e;

  if (pl.splits > 1) {
    // all splits of a unit wait for one another: they must be resident together
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    return launch(attn_tc_kernel, dim3(pl.splits, pl.n_pairs, p.batch * p.hkv), dim3(kThreads),
                  kSmemBytes, s, attr, 1, tq, tk, tv, a);
  }
  return launch(attn_tc_kernel, dim3(pl.units), dim3(kThreads), kSmemBytes, s, nullptr, 0, tq, tk, tv,
                a);
}

}  // namespace ltd

#ifdef LTD_TRACE
extern "C" int ltd_attn_trace_read(unsigned long long* host, int n) {
  return cudaMemcpyFromSymbol(host, ltd::g_attn_trace, sizeof(unsigned long long) * n) == cudaSuccess
             ? 0
             : 1;
}
#endif
