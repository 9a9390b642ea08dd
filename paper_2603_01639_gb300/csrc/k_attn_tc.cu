// Tensor-core tree attention (LTD section 3.2, "Draft Tree Verification";
// SpecInfer-style tree mask) for bf16 and head_dim 128 on sm_103a.
//
// Work unit: one 128-row tile of the query rows of one KV head of one
// sequence (row r = slot * G + g, so the G query heads of a KV head share
// every K/V byte), over one split of that head's keys.  The split's 128-key
// chunks go to two streams, even chunks to stream 0 and odd chunks to stream
// 1; each stream has its own S and O in tensor memory and its own running
// max and sum, so one stream's softmax runs while the tensor core works on
// the other's chunk, and the two are merged once at the end.
//   warp 0      TMA: the Q tile, then K chunks into a three-stage ring
//               (128-byte swizzle); Q and the first K chunk are issued
//               before the sequence's context length is read;
//   warp 1      tcgen05.mma: S_x = Q K_j^T into tensor memory, then
//               O_x += P_x V_j with P_x read from tensor memory, issued in
//               the order S(0), S(1), PV(0), S(2), PV(1), S(3), ...; the
//               waits of a pair PV(j), S(j+2) all come before its first MMA,
//               so the pair goes out back to back;
//   warp 2      TMA: V chunks into a three-stage ring;
//   warps 4-7   softmax of stream 0, warps 8-11 of stream 1, one thread per
//               row (= tensor-memory lane) with the row's 128 scores in
//               registers: the prefix + ancestor mask, then P = 2^(s - m)
//               against the stream's running max m, computed before the
//               chunk's own max is known and redone only for a warp in which
//               some row's max grew by more than 2^8 (S is still in tensor
//               memory then); O is rescaled only in that case.  P is written
//               as bf16 over S's columns.
// Tensor memory (512 columns): S_0 | S_1 | O_0 | O_1.
//
// Two launch shapes:
//  - one split per unit (at least as many units as SMs): each CTA writes
//    O / l straight to the output, and CTAs take the units longest first
//    (every CTA ranks the (sequence, tile) groups by their chunk counts from
//    ctx and N), so the long sequences of a ragged batch start early;
//  - several splits per unit (fewer units than SMs): a cooperative launch,
//    so every CTA is resident at once.  Each split writes its rows' O / l
//    (bf16) and log2-sum-exp to the workspace and arrives on its unit's
//    counter; when all splits have arrived, split s combines rows
//    [s R, s R + R) of the unit with loads straight from L2 into registers
//    and writes them; the last split to leave resets the unit's counters.
// Every wait is bounded (mbarrier waits, which sleep in hardware between
// tries, and the counter spin): on timeout a CTA flags LTD_DEVERR_TIMEOUT,
// drains its own TMA loads and MMAs, still arrives and departs on its
// counter, frees its tensor memory and returns.
#include <mutex>
#include <type_traits>

#include "ltd_common.cuh"
#include "ltd_internal.h"
#include "tc_util.cuh"

namespace ltd {

namespace {

constexpr int kBM = 128;  // rows per tile = TMEM lanes
constexpr int kBN = 128;  // keys per chunk
constexpr int kD = 128;
constexpr int kStages = 3;             // K ring and V ring depth
constexpr int kThreads = 384;          // K TMA, MMA, V TMA, idle, 8 softmax warps
constexpr int kMaxSplits = 64;
constexpr int kMaxGroups = 1024;       // (sequence, tile) groups ranked on the device
constexpr int kCombineBatch = 16;      // splits whose partials one combining thread has in flight
constexpr uint32_t kHalf = 16384;      // 128 rows x 128 bytes
constexpr uint32_t kTile = 2 * kHalf;  // 128 x 128 bf16
constexpr uint32_t kOffQ = 0;
constexpr uint32_t kOffK = kOffQ + kTile;             // three stages
constexpr uint32_t kOffV = kOffK + kStages * kTile;   // three stages
constexpr uint32_t kOffBar = kOffV + kStages * kTile;
constexpr uint32_t kOffHolder = kOffBar + 24 * 8;
constexpr uint32_t kSmemBytes = kOffHolder + 16 + 1024;  // + alignment slack
// Regions reused once they are free (after the last MMA, or before any load):
constexpr uint32_t kOffCost = kOffV + 2 * kTile;       // [kMaxGroups] int, ranking only
constexpr uint32_t kOffOrder = kOffCost + kMaxGroups * 4;
constexpr uint32_t kOffML = kOffK + 1024;              // [2][128] (m, l) of each stream
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kRowBytes = kD * 2;  // one bf16 output / partial row
// P may grow to 2^8 before a row's running max is raised: bf16 bits of 2^8
constexpr uint32_t kPMaxBits = 0x4380u;

static_assert(kSmemBytes <= 232448, "shared memory over the per-block limit");
static_assert(kOffOrder + kMaxGroups * 4 <= kOffV + kStages * kTile, "ranking arrays overflow");

// barrier indices
constexpr int QFULL = 0;
constexpr int KFULL = 1;    // + stage
constexpr int VFULL = 4;    // + stage
constexpr int KEMPTY = 7;   // + stage
constexpr int VEMPTY = 10;  // + stage
constexpr int SFULL = 13;   // + stream
constexpr int PFULL = 15;   // + stream
constexpr int FIN = 17;

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
  int32_t splits, n_tiles, lpt;
  int32_t nch_h;  // host bound on chunks per sequence: ceil((max_ctx + n_max) / 128)
  int32_t rs;     // rows combined per split: ceil(128 / splits)
  const int32_t* ctx;
  const int32_t* n_verify;
  const uint32_t* mask;
  float scale_log2;
  __nv_bfloat16* out;
  uint8_t* part_o;  // [unit][split][16 chunks][128 rows][16 B] O / l, bf16 (splits > 1)
  float* part_l;    // [unit][split][128] log2-sum-exp
  uint32_t* sync;   // [unit][2] arrive, depart
  const uint8_t* next_k;  // the next call's caches: L2 prefetch targets (or null)
  const uint8_t* next_v;
  uint32_t* err;
  // K and V through one tensor map when both caches fit one 4-D map (the
  // fourth coordinate picks the cache), else one map each
  int32_t kv_one, kv_wk, kv_wv;
  // the split counter's wait: its limit, and arrivals awaited beyond the
  // unit's splits (a test hook; 0 in normal calls, so the wait completes)
  uint64_t spin_limit_ns;
  uint32_t extra_arrivals;
};

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&v);
}

// Visibility of keys kk0 .. kk0+31 for one row as a 32-bit mask: keys below
// ctx are the prefix (always visible), key ctx + j is verified slot j (bit j
// of the row's ancestor mask), keys from key_hi on are outside this split.
// `lo` and `hi` are the mask words holding slots (kk0 - ctx) >> 5 and the one
// after (0 outside the mask), `sh` = (kk0 - ctx) & 31.
__device__ __forceinline__ uint32_t low_bits(int n) {
  return n <= 0 ? 0u : (n >= 32 ? 0xFFFFFFFFu : ((1u << n) - 1u));
}
__device__ __forceinline__ uint32_t visible32(int kk0, int ctx, int key_hi, uint32_t lo, uint32_t hi,
                                              int sh) {
  return low_bits(key_hi - kk0) & (low_bits(ctx - kk0) | __funnelshift_r(lo, hi, sh));
}

__device__ __forceinline__ bool seq_ok(const TcArgs& a, int ctx, int N) {
  return N >= 1 && N <= a.n_max && ctx >= 0 && ctx <= a.max_ctx && ctx + N <= a.s_cap;
}

__device__ __forceinline__ uint4 ld_cg_v4(const void* p) {
  uint4 v;
  asm volatile("ld.global.cg.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}
__device__ __forceinline__ float ld_cg_f32(const float* p) {
  float v;
  asm volatile("ld.global.cg.f32 %0, [%1];" : "=f"(v) : "l"(p));
  return v;
}

template <int N>
using Int = std::integral_constant<int, N>;

__global__ void __launch_bounds__(kThreads, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tq, const __grid_constant__ CUtensorMap tk,
                   const __grid_constant__ CUtensorMap tv, const TcArgs a) {
  extern __shared__ uint8_t smem_raw[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) TRACE(0);
  const uint32_t raw = tc::smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  uint32_t* holder = reinterpret_cast<uint32_t*>(gbase + kOffHolder);
  auto bar = [&](int i) { return base + kOffBar + 8u * i; };
  const int S = a.splits;

  if (tid == 0) {
    tc::tma_prefetch(&tq);
    tc::tma_prefetch(&tk);
    if (!a.kv_one) tc::tma_prefetch(&tv);
    TRACE(42);
    tc::mbar_init(bar(QFULL), 1);
    for (int s = 0; s < kStages; ++s) {
      tc::mbar_init(bar(KFULL + s), 1);
      tc::mbar_init(bar(VFULL + s), 1);
      tc::mbar_init(bar(KEMPTY + s), 1);
      tc::mbar_init(bar(VEMPTY + s), 1);
    }
    for (int x = 0; x < 2; ++x) {
      tc::mbar_init(bar(SFULL + x), 1);
      tc::mbar_init(bar(PFULL + x), 128);
    }
    tc::mbar_init(bar(FIN), 1);
    tc::mbar_init_fence();
    TRACE(19);
  }
  // everything above touches only shared memory and this launch's
  // parameters; what follows may read another kernel's output
  grid_wait();
  trigger_dependents();
  if (tid == 0) TRACE(43);

  // ------------------------------------------------------ which unit
  int split = 0, tile, b, kvh;
  if (S > 1) {
    split = blockIdx.x;
    tile = blockIdx.y;
    b = blockIdx.z / a.hkv;
    kvh = blockIdx.z % a.hkv;
  } else {
    const int i = blockIdx.x;
    int g = i / a.hkv;
    kvh = i % a.hkv;
    if (a.lpt) {
      // rank every (sequence, tile) group by its work, largest first (ties
      // to the lower group, so the tiles of one sequence, which read the
      // same K/V, stay together), and take the group at this CTA's rank;
      // bad sequences rank last and flag on their own CTAs
      int* cost = reinterpret_cast<int*>(gbase + kOffCost);
      int* order = reinterpret_cast<int*>(gbase + kOffOrder);
      const int groups = a.batch * a.n_tiles;
      for (int gi = tid; gi < groups; gi += kThreads) {
        const int bb = gi / a.n_tiles, tt = gi % a.n_tiles;
        const int c = a.ctx[bb], n = a.n_verify[bb];
        int w = 0;
        if (seq_ok(a, c, n) && n * a.G > tt * kBM) w = (c + n + kBN - 1) / kBN;
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
    b = g / a.n_tiles;
    tile = g % a.n_tiles;
  }

  // Keys are split by the host bound on the chunk count, so a split knows
  // its first chunk before reading ctx and N: the loads of Q and of the
  // first K chunk go out at once (a chunk past this sequence's end is
  // drained and ignored).  The other chunks wait for the setup below.
  const int cs = split * a.nch_h / S, ce = (split + 1) * a.nch_h / S;
  const int kvrow = b * a.hkv + kvh;
  const int row0 = tile * kBM;
  int nk_issued[kStages] = {0, 0, 0};
  bool q_issued = false;
  auto issue_k = [&](int j) {
    const int st = j % kStages;
    tc::mbar_expect_tx(bar(KFULL + st), kTile);
    for (int h = 0; h < 2; ++h)
      tc::tma_load_4d(base + kOffK + st * kTile + h * kHalf, &tk, bar(KFULL + st), h * 64,
                      (cs + j) * kBN, kvrow, a.kv_wk);
    ++nk_issued[st];
  };
  auto issue_first = [&]() {
    tc::mbar_expect_tx(bar(QFULL), kTile);
    const int qrow = b * a.n_max + row0 / a.G;
    for (int h = 0; h < 2; ++h)
      tc::tma_load_3d(base + kOffQ + h * kHalf, &tq, bar(QFULL), h * 64, kvh * a.G, qrow);
    q_issued = true;
    TRACE(20);
    if (ce - cs > 0) issue_k(0);
    TRACE(17);
  };
  // every K load (and Q) this thread issued lands before the CTA leaves or
  // reuses shared memory; at most one load per stage is outstanding
  auto drain_k = [&]() {
    if (q_issued) tc::mbar_wait_sleep(bar(QFULL), 0);
    for (int st = 0; st < kStages; ++st)
      if (nk_issued[st] > 0) tc::mbar_wait_sleep(bar(KFULL + st), (nk_issued[st] - 1) & 1);
  };
  if (tid == 0 && !a.lpt) issue_first();

  // Everything a CTA returns early on is shared by all splits of its unit.
  const int ctx = a.ctx[b];
  const int N = a.n_verify[b];
  const int M = N * a.G;
  if (tid == 0) TRACE(21);
  if (!seq_ok(a, ctx, N) || row0 >= M) {
    if (tid == 0) {
      if (!seq_ok(a, ctx, N) && split == 0 && tile == 0 && kvh == 0)
        flag_error(a.err, (N < 1 || N > a.n_max) ? LTD_DEVERR_NVERIFY : LTD_DEVERR_CTX);
      drain_k();
    }
    return;
  }
  const int nk = ctx + N;
  const int nch = (nk + kBN - 1) / kBN;
  const int nc = max(0, min(ce, nch) - cs);
  const int key_lo = cs * kBN, key_hi = min(ce * kBN, nk);

  if (tid == 0 && a.lpt) issue_first();
  if (warp == 1) {
    tc::tmem_alloc(tc::smem_u32(holder), kTmemCols);
    tc::tmem_relinquish();
  }
  // softmax threads (warps 4-11): stream x, TMEM lane lrow = row of the tile
  const bool smx = warp >= 4;
  const int x = (warp - 4) >> 2;
  const int lrow = 32 * (warp & 3) + lane;
  const int R = row0 + lrow;
  const bool row_ok = smx && R < M;
  // the row's ancestor-mask words, read where a chunk holds verified keys
  const uint32_t* mbits =
      a.mask + (static_cast<int64_t>(b) * a.n_max + min(R / a.G, a.n_max - 1)) * a.W32;
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = holder[0];
  if (tid == 0) TRACE(1);
  bool ok = true;
  float m = -CUDART_INF_F, l = 0.f;  // the stream's running max (log2 units) and sum

  if (warp == 0) {
    // ------------------------------------------------------- K producer
    if (lane == 0) {
      for (int j = 1; j < nc && j < kStages; ++j) issue_k(j);
      for (int j = kStages; j < nc && ok; ++j) {
        ok = tc::mbar_wait_sleep(bar(KEMPTY + j % kStages), ((j / kStages) - 1) & 1);
        if (ok) issue_k(j);
      }
      drain_k();
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
      TRACE(31);
    }
  } else if (warp == 2) {
    // ------------------------------------------------------- V producer
    if (lane == 0) {
      int nv_issued[kStages] = {0, 0, 0};
      auto issue_v = [&](int j) {
        const int st = j % kStages;
        tc::mbar_expect_tx(bar(VFULL + st), kTile);
        for (int h = 0; h < 2; ++h)
          tc::tma_load_4d(base + kOffV + st * kTile + h * kHalf, a.kv_one ? &tk : &tv,
                          bar(VFULL + st), h * 64, (cs + j) * kBN, kvrow, a.kv_wv);
        ++nv_issued[st];
      };
      for (int j = 0; j < nc && j < kStages; ++j) issue_v(j);
      for (int j = kStages; j < nc && ok; ++j) {
        ok = tc::mbar_wait_sleep(bar(VEMPTY + j % kStages), ((j / kStages) - 1) & 1);
        if (ok) issue_v(j);
      }
      for (int st = 0; st < kStages; ++st)
        if (nv_issued[st] > 0) tc::mbar_wait_sleep(bar(VFULL + st), (nv_issued[st] - 1) & 1);
      if (!ok) flag_error(a.err, LTD_DEVERR_TIMEOUT);
    }
  } else if (warp == 1) {
    // ----------------------------------------------------------------- MMA
    if (lane == 0 && nc > 0) {
      const uint32_t id_s = tc::idesc_bf16(kBM, kBN, false);
      const uint32_t id_o = tc::idesc_bf16(kBM, kD, true);
      // Three base descriptors; the others differ by constant offsets (in
      // 16-byte units) for the K slice and the ring stage: K-major slice ks
      // at (ks / 4) * kHalf + (ks % 4) * 32 bytes, MN-major slice ks of V 16
      // rows of 128 bytes on.
      const uint64_t dq0 = tc::sdesc_sw128(base + kOffQ, 16, 1024);
      const uint64_t dk0 = tc::sdesc_sw128(base + kOffK, 16, 1024);
      const uint64_t dv0 = tc::sdesc_sw128(base + kOffV, kHalf, 1024);
      if (nc <= 4) {
        // a short split: a rolled loop, stage descriptors by adds per chunk
        // (this thread runs its issue code cold, and a short split runs it
        // only a few times)
        auto koff = [](int ks) { return static_cast<uint64_t>((ks >> 2) * (kHalf >> 4) + (ks & 3) * 2); };
        auto issue_s = [&](int x_, int st) {
          const uint64_t k = dk0 + static_cast<uint64_t>(st) * (kTile >> 4);
          const uint32_t d = tmem + x_ * kBN;
#pragma unroll
          for (int ks = 0; ks < 8; ++ks) tc::mma_bf16(d, dq0 + koff(ks), k + koff(ks), id_s, ks > 0 ? 1u : 0u);
        };
        auto issue_pv = [&](int x_, int st, uint32_t acc) {
          const uint64_t v = dv0 + static_cast<uint64_t>(st) * (kTile >> 4);
          const uint32_t d = tmem + 2 * kBN + x_ * kD, pa = tmem + x_ * kBN;
#pragma unroll
          for (int ks = 0; ks < 8; ++ks)
            tc::mma_bf16_ts(d, pa + 8 * ks, v + static_cast<uint64_t>(ks * (2048 >> 4)), id_o, ks > 0 ? 1u : acc);
        };
        ok = tc::mbar_wait_sleep(bar(QFULL), 0);
        TRACE(2);
        // S(0) and S(1) into S_0 and S_1, then per chunk j (stream j & 1, ring
        // stage j % 3, ring use j / 3): PV(j), then S(j + 2) into the same
        // stream
        for (int j = 0; j < 2 && j < nc && ok; ++j) {
          ok = tc::mbar_wait_sleep(bar(KFULL + j), 0);
          if (!ok) break;
          tc::fence_after_sync();
          issue_s(j, j);
          tc::mma_commit(bar(SFULL + j));
          tc::mma_commit(bar(KEMPTY + j));
          if (j == 0) TRACE(3);
        }
        for (int j = 0; j < nc && ok; ++j) {
          const int xs = j & 1, st = j % kStages, st2 = (j + 2) % kStages;
          const bool more = j + 2 < nc;
          // every wait before the first MMA of the pair, the one that
          // usually blocks (P) last: a wait between MMA groups is a bubble
          // in the tensor pipe even when its phase has completed
          if (more) ok = tc::mbar_wait_sleep(bar(KFULL + st2), ((j + 2) / kStages) & 1);
          if (ok) ok = tc::mbar_wait_sleep(bar(VFULL + st), (j / kStages) & 1);
          if (ok) ok = tc::mbar_wait_sleep(bar(PFULL + xs), (j >> 1) & 1);
          if (!ok) break;
          tc::fence_after_sync();
          issue_pv(xs, st, j >= 2 ? 1u : 0u);
          tc::mma_commit(bar(VEMPTY + st));
          if (more) {
            issue_s(xs, st2);
            tc::mma_commit(bar(SFULL + xs));
            tc::mma_commit(bar(KEMPTY + st2));
          }
        }
      } else {
        // a long split: the loop unrolled over six chunks, so stages and
        // descriptors are compile-time choices
        // every descriptor of the loop, from the three bases by adds (held in
        // registers: the issue loop below is MMA instructions and waits only)
        uint64_t dq[8], dk[kStages][8], dv[kStages][8];
#pragma unroll
        for (int ks = 0; ks < 8; ++ks) {
          const uint64_t ko = static_cast<uint64_t>((ks >> 2) * (kHalf >> 4) + (ks & 3) * 2);
          dq[ks] = dq0 + ko;
#pragma unroll
          for (int st = 0; st < kStages; ++st) {
            dk[st][ks] = dk0 + static_cast<uint64_t>(st * (kTile >> 4)) + ko;
            dv[st][ks] = dv0 + static_cast<uint64_t>(st * (kTile >> 4) + ks * (2048 >> 4));
          }
        }
        // (x and st are compile-time constants at every call)
        auto issue_s = [&](int x_, int st) {
#pragma unroll
          for (int ks = 0; ks < 8; ++ks)
            tc::mma_bf16(tmem + x_ * kBN, dq[ks], dk[st][ks], id_s, ks > 0 ? 1u : 0u);
        };
        auto issue_pv = [&](int x_, int st, uint32_t acc) {
#pragma unroll
          for (int ks = 0; ks < 8; ++ks)
            tc::mma_bf16_ts(tmem + 2 * kBN + x_ * kD, tmem + x_ * kBN + 8 * ks, dv[st][ks], id_o,
                            ks > 0 ? 1u : acc);
        };
        ok = tc::mbar_wait_sleep(bar(QFULL), 0);
        TRACE(2);
        // S(0) and S(1) into S_0 and S_1, then chunk j = 6 i + r (stream r & 1,
        // ring stage r % 3, ring use j / 3, whose parity is (r / 3) & 1): PV(j),
        // then S(j + 2) into the same stream; stages are compile-time constants
        if (ok) ok = tc::mbar_wait_sleep(bar(KFULL + 0), 0);
        if (ok) {
          tc::fence_after_sync();
          issue_s(0, 0);
          tc::mma_commit(bar(SFULL + 0));
          tc::mma_commit(bar(KEMPTY + 0));
        }
        TRACE(3);
        if (ok && nc > 1) {
          ok = tc::mbar_wait_sleep(bar(KFULL + 1), 0);
          if (ok) {
            tc::fence_after_sync();
            issue_s(1, 1);
            tc::mma_commit(bar(SFULL + 1));
            tc::mma_commit(bar(KEMPTY + 1));
          }
        }
        auto step = [&](int j, auto R_) -> bool {
          constexpr int r = decltype(R_)::value;
          constexpr int xs = r & 1, st = r % kStages, st2 = (r + 2) % kStages;
          const bool more = j + 2 < nc;
          // (every wait before the pair's first MMA, P last, as above)
          bool k = !more || tc::mbar_wait_sleep(bar(KFULL + st2), ((r + 2) / kStages) & 1);
          if (k) k = tc::mbar_wait_sleep(bar(VFULL + st), (r / kStages) & 1);
          if (k) k = tc::mbar_wait_sleep(bar(PFULL + xs), (j >> 1) & 1);
          if (!k) return false;
          tc::fence_after_sync();
          issue_pv(xs, st, j >= 2 ? 1u : 0u);
          tc::mma_commit(bar(VEMPTY + st));
          if (more) {
            issue_s(xs, st2);
            tc::mma_commit(bar(SFULL + xs));
            tc::mma_commit(bar(KEMPTY + st2));
          }
          return true;
        };
        for (int j = 0; j < nc && ok; j += 6) {
          ok = step(j, Int<0>{});
          if (ok && j + 1 < nc) ok = step(j + 1, Int<1>{});
          if (ok && j + 2 < nc) ok = step(j + 2, Int<2>{});
          if (ok && j + 3 < nc) ok = step(j + 3, Int<3>{});
          if (ok && j + 4 < nc) ok = step(j + 4, Int<4>{});
          if (ok && j + 5 < nc) ok = step(j + 5, Int<5>{});
        }
      }
      TRACE(22);
      // every MMA of this CTA completes before tensor memory is read or freed
      tc::mma_commit(bar(FIN));
      tc::mbar_wait_sleep(bar(FIN), 0);
      if (!ok) flag_error(a.err, LTD_DEVERR_TIMEOUT);
      TRACE(23);
    }
#ifdef LTD_TRACE
  } else if (warp == 3) {
    // (trace builds only) the idle warp observes when the first loads land
    if (lane == 0) {
      if (tc::mbar_wait_sleep(bar(QFULL), 0)) TRACE(24);
      if (nc > 0 && tc::mbar_wait_sleep(bar(KFULL + 0), 0)) TRACE(25);
      if (nc > 0 && tc::mbar_wait_sleep(bar(VFULL + 0), 0)) TRACE(26);
      if (nc > 1 && tc::mbar_wait_sleep(bar(KFULL + 1), 0)) TRACE(27);
      if (nc > 1 && tc::mbar_wait_sleep(bar(VFULL + 1), 0)) TRACE(28);
      if (nc > 2 && tc::mbar_wait_sleep(bar(KFULL + 2), 0)) TRACE(29);
      if (nc > 2 && tc::mbar_wait_sleep(bar(VFULL + 2), 0)) TRACE(30);
    }
#endif
  } else if (smx && x < nc) {
    // ------------------------------------------------------------- softmax
    const uint32_t lane_off = (32u * (warp & 3)) << 16;
    const uint32_t t_s = tmem + x * kBN + lane_off;
    const uint32_t t_o = tmem + 2 * kBN + x * kD + lane_off;
    const int vis_all_below = min(ctx, key_hi);  // keys below this are all visible
    const float sl2 = a.scale_log2;
    const int w32 = a.W32;
    const bool tr = (tid & 127) == 0;
    for (int j = x; j < nc; j += 2) {
      const int kbase = key_lo + j * kBN;
      const bool all_vis = row_ok && kbase + kBN <= vis_all_below;
      // A chunk that holds verified keys needs five of the row's mask words
      // (its four 32-key windows and the word after), read from L2 (the
      // mask is another kernel's output) before the wait below, so their
      // latency hides behind it.
      uint32_t mw5[5] = {0u, 0u, 0u, 0u, 0u};
      const int js = kbase - ctx, w0 = js >> 5;  // floor division
      if (row_ok && !all_vis) {
#pragma unroll
        for (int t = 0; t < 5; ++t)
          if (w0 + t >= 0 && w0 + t < w32) mw5[t] = __ldcg(mbits + w0 + t);
      }
      ok = tc::mbar_wait_sleep(bar(SFULL + x), (j >> 1) & 1);
      ok = __all_sync(0xFFFFFFFFu, ok);
      if (tr && j < 4) TRACE(4 + 2 * j);
      if (!ok) break;
      tc::fence_after_sync();
      // P against the stream's running max m (a row without one yet first
      // takes this chunk's max); the chunk's own max is tracked on the way
      // and, if it exceeds the reference by more than 2^8 in some row of the
      // warp, the warp re-derives P from S, still intact in tensor memory, 32
      // columns at a time.
      tc::Frag128 f;
      float mref = m;
      float2 ls2 = make_float2(0.f, 0.f);
      uint32_t vq[4] = {0xFFFFFFFFu, 0xFFFFFFFFu, 0xFFFFFFFFu, 0xFFFFFFFFu};
      if (!all_vis) {
#pragma unroll
        for (int qq = 0; qq < 4; ++qq)
          vq[qq] = row_ok ? visible32(kbase + 32 * qq, ctx, key_hi, mw5[qq], mw5[qq + 1], js & 31) : 0u;
      }
      __syncwarp();  // the load below is warp-collective; the branch above is per row
      tc::tmem_ld128_sync(t_s, f);
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
      // S(j) was issued after PV(j - 2) of this stream, so O_x is stable here
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
      if (kbase + kBN > key_hi) {
        // Keys from key_hi on may hold anything in the cache, even NaN: P is
        // 0 there, but 0 * NaN is not, so this stream's threads clear those V
        // rows (both 64-dim halves) before PV reads this stage.
        const int st = j % kStages;
        // (a failed wait is flagged; the MMA thread times out on the same stage)
        if (!__all_sync(0xFFFFFFFFu, tc::mbar_wait_sleep(bar(VFULL + st), (j / kStages) & 1)) && lane == 0)
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
      tc::fence_before_sync();
      tc::mbar_arrive(bar(PFULL + x));
      if (tr && j < 4) TRACE(5 + 2 * j);
    }
    if (!ok && lane == 0) flag_error(a.err, LTD_DEVERR_TIMEOUT);
    if (tr) TRACE(12 + x);
  }

  // --------------------------------------------------------- epilogue
  // The producers have drained every load and the MMA thread has seen the
  // last MMA complete before this barrier; after it, the K ring holds the
  // two streams' (m, l).
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  if (tid == 0) TRACE(14);
  float2* ml = reinterpret_cast<float2*>(gbase + kOffML);
  if (smx) ml[x * kBM + lrow] = make_float2(m, l);
  __syncthreads();
  if (tid == 0) TRACE(32);
  const int unit = (b * a.hkv + kvh) * a.n_tiles + tile;
  const int Mv = min(kBM, M - row0);
  const int Rp = (Mv + 7) & ~7;  // rows of a partial block (16-byte chunk-major)
  const int64_t pb = static_cast<int64_t>(unit) * S + split;
  // Merge the two streams: stream x's thread of a row writes columns
  // 64 x .. 64 x + 63 of O / l, straight from registers to the output (one
  // split), or (several splits) into shared memory over Q's region,
  // chunk-major ([16-byte chunk][row], so a warp's stores are contiguous),
  // with the row's log2-sum-exp over the K ring; one bulk copy then stores
  // the block as this split's partial.  tcgen05.ld is warp-collective: the
  // loads are taken by whole warps (nc is uniform), the writes per row.
  if (smx) {
    const float2 me = ml[lrow], mo = ml[kBM + lrow];
    const float mm = fmaxf(me.x, mo.x);
    const float a0 = mm == -CUDART_INF_F ? 0.f : tc::ex2(me.x - mm);
    const float a1 = mm == -CUDART_INF_F ? 0.f : tc::ex2(mo.x - mm);
    const float L = me.y * a0 + mo.y * a1;
    const bool have = L > 0.f;
    const float inv = have ? 1.f / L : 0.f;
    const float w0 = a0 * inv, w1 = a1 * inv;
    const uint32_t lane_off = (32u * (warp & 3)) << 16;
    const bool ld0 = nc > 0, ld1 = nc > 1;
    tc::Frag64 o0, o1;
    if (ld0) tc::tmem_ld64_sync(tmem + 2 * kBN + 0 * kD + 64 * x + lane_off, o0);
    if (ld1) tc::tmem_ld64_sync(tmem + 2 * kBN + 1 * kD + 64 * x + lane_off, o1);
    if (row_ok) {
      uint4* dst;
      int64_t step;
      if (S == 1) {
        const int slot = R / a.G, g = R % a.G;
        dst = reinterpret_cast<uint4*>(a.out + ((static_cast<int64_t>(b) * a.n_max + slot) * a.hq +
                                                kvh * a.G + g) * kD) + 8 * x;
        step = 1;
      } else {
        // staged chunk-major over Q's region, stored below with one bulk copy
        dst = reinterpret_cast<uint4*>(gbase + kOffQ) + (8 * x) * Rp + lrow;
        step = Rp;
      }
#pragma unroll
      for (int c = 0; c < 8; ++c) {
        float v[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          float s = 0.f;
          if (have && ld0) s = __uint_as_float(o0.r[8 * c + e]) * w0;
          if (have && ld1) s = fmaf(__uint_as_float(o1.r[8 * c + e]), w1, s);
          v[e] = s;
        }
        uint4 w;
        w.x = pack_bf16(v[0], v[1]);
        w.y = pack_bf16(v[2], v[3]);
        w.z = pack_bf16(v[4], v[5]);
        w.w = pack_bf16(v[6], v[7]);
        dst[c * step] = w;
      }
      if (S > 1 && x == 0)
        reinterpret_cast<float*>(gbase + kOffK)[lrow] = have ? mm + __log2f(L) : -CUDART_INF_F;
    }
  }
  tc::fence_smem_async();  // the staging is read by bulk copies
  tc::fence_before_sync();
  __syncthreads();
  if (tid == 0) TRACE(15);
  if (warp == 1) {
    __syncwarp();
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, kTmemCols);
  }
  if (S == 1) return;

  // ------------------------------------- combine the splits (S > 1 only)
  // Each split stores its staged block and sums with one bulk copy each and
  // waits for their completion before it arrives on its unit's counter.
  // (Plain stores from registers, each thread fencing before the CTA
  // barrier and one thread releasing the counter, were measured to let the
  // owners read incomplete partials.)  Rows [o rs, o rs + rs) of a unit are
  // combined by its split o, every thread loading one 16-byte chunk of one
  // row from every split straight into registers.
  uint32_t* arrive = a.sync + 2 * unit;
  uint32_t* depart = arrive + 1;
  if (tid == 0) {
    tc::bulk_s2g(a.part_o + pb * 16 * kBM * 16, base + kOffQ, 16 * Rp * 16);
    tc::bulk_s2g(a.part_l + pb * kBM, base + kOffK, Rp * 4);
    tc::bulk_commit();
    tc::bulk_wait_all();
    tc::fence_proxy_async_global();
    tc::red_add_release_gpu(arrive, 1u);
    TRACE(34);
    const uint32_t quorum = static_cast<uint32_t>(S) + a.extra_arrivals;
    bool got = tc::ld_acquire_gpu(arrive) >= quorum;
    if (!got) {
      const uint64_t t0 = tc::globaltimer();
      while (!got) {
        __nanosleep(32);
        got = tc::ld_acquire_gpu(arrive) >= quorum;
        if (!got && tc::globaltimer() - t0 > a.spin_limit_ns) break;
      }
    }
    if (!got) flag_error(a.err, LTD_DEVERR_TIMEOUT);
    holder[1] = got ? 1u : 0u;
    TRACE(16);
  }
  __syncthreads();
  const int Rs = a.rs;
  const int r_lo = split * Rs;
  const int nrows = max(0, min(Mv, r_lo + Rs) - r_lo);
  // the acquire above (ordered by the barrier) makes the other splits'
  // stores visible; .cg loads read them from L2
  if (tid == 0) TRACE(35);
  for (int idx = tid; holder[1] != 0u && idx < nrows * 16; idx += kThreads) {
    // consecutive threads take consecutive rows of one chunk (contiguous)
    const int c = idx / nrows, r = r_lo + idx % nrows;
    const int64_t ub = static_cast<int64_t>(unit) * S;
    const uint4* src = reinterpret_cast<const uint4*>(a.part_o) + ub * 16 * kBM + c * Rp + r;
    const float* lsrc = a.part_l + ub * kBM + r;
    float mx = -CUDART_INF_F, L = 0.f;
    float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    for (int p0 = 0; p0 < S; p0 += kCombineBatch) {
      uint4 v[kCombineBatch];
      float ls[kCombineBatch];
#pragma unroll
      for (int u = 0; u < kCombineBatch; ++u) {
        const int p = p0 + u;
        ls[u] = p < S ? ld_cg_f32(lsrc + static_cast<int64_t>(p) * kBM) : -CUDART_INF_F;
        v[u] = p < S ? ld_cg_v4(src + static_cast<int64_t>(p) * 16 * kBM) : make_uint4(0u, 0u, 0u, 0u);
      }
      float bm = mx;
#pragma unroll
      for (int u = 0; u < kCombineBatch; ++u) bm = fmaxf(bm, ls[u]);
      if (bm > -CUDART_INF_F) {
        const float sc = tc::ex2(mx - bm);  // 0 while mx is -inf
        L *= sc;
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[e] *= sc;
#pragma unroll
        for (int u = 0; u < kCombineBatch; ++u) {
          const float w = tc::ex2(ls[u] - bm);  // 0 for a split without keys
          L += w;
          const uint32_t ev[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
#pragma unroll
          for (int t = 0; t < 4; ++t) {
            acc[2 * t] = fmaf(w, __uint_as_float(ev[t] << 16), acc[2 * t]);
            acc[2 * t + 1] = fmaf(w, __uint_as_float(ev[t] & 0xFFFF0000u), acc[2 * t + 1]);
          }
        }
        mx = bm;
      }
    }
    if (idx == 0) TRACE(36);
    const float inv = L > 0.f ? 1.f / L : 0.f;
    const int Rr = row0 + r;
    const int slot = Rr / a.G, g = Rr % a.G;
    uint4 w;
    w.x = pack_bf16(acc[0] * inv, acc[1] * inv);
    w.y = pack_bf16(acc[2] * inv, acc[3] * inv);
    w.z = pack_bf16(acc[4] * inv, acc[5] * inv);
    w.w = pack_bf16(acc[6] * inv, acc[7] * inv);
    reinterpret_cast<uint4*>(a.out + ((static_cast<int64_t>(b) * a.n_max + slot) * a.hq +
                                      kvh * a.G + g) * kD)[c] = w;
  }
  __syncthreads();
  if (tid == 0) {
    TRACE(18);
    // every split of this unit has passed its spin once all have departed
    const uint32_t d = atomicAdd(depart, 1u);
    if (d == static_cast<uint32_t>(S) - 1u) {
      atomicExch(arrive, 0u);
      atomicExch(depart, 0u);
    }
  }
}

struct Plan {
  int n_tiles, splits, units, lpt, nch, rs;
};


// The split counter's wait settings for later launches (test hook).
std::mutex g_hook_mu;
AttnWaitHook g_hook{};

// Units = (sequence, KV head, tile).  With fewer units than SMs each unit's
// keys are cut into the fewest splits that give the shortest longest split,
// at most SMs / units of them, so all CTAs fit one wave.
Plan plan(int32_t batch, int32_t hq, int32_t hkv, int32_t n_max, int32_t max_ctx) {
  const int G = hq / hkv;
  Plan p{};
  p.n_tiles = (n_max * G + kBM - 1) / kBM;
  const int64_t units = static_cast<int64_t>(batch) * hkv * p.n_tiles;
  p.units = static_cast<int>(units);
  const int nch = (max_ctx + n_max + kBN - 1) / kBN;
  const int sms = device_sm_count();
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
  p.lpt = (p.splits == 1 && static_cast<int64_t>(batch) * p.n_tiles <= kMaxGroups) ? 1 : 0;
  p.nch = nch;
  p.rs = (kBM + p.splits - 1) / p.splits;
  return p;
}

size_t align256(size_t n) { return (n + 255) / 256 * 256; }

struct WsLayout {
  size_t part_o, part_l, sync, total;
};
WsLayout ws_layout(const Plan& pl) {
  WsLayout w{};
  if (pl.splits <= 1) return w;
  // [unit][split][128] rows
  const size_t rows = static_cast<size_t>(pl.units) * pl.splits * kBM;
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

// Streaming multiprocessors of the current device (152 if it cannot be asked).
int device_sm_count() {
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

void set_attn_wait_hook(const AttnWaitHook& h) {
  std::lock_guard<std::mutex> lock(g_hook_mu);
  g_hook = h;
}
AttnWaitHook attn_wait_hook() {
  std::lock_guard<std::mutex> lock(g_hook_mu);
  return g_hook;
}

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
  a.n_tiles = pl.n_tiles;
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
  {
    const AttnWaitHook h = attn_wait_hook();
    a.spin_limit_ns = h.limit_ns != 0 ? h.limit_ns : tc::kWaitLimitNs;
    a.extra_arrivals = h.extra_arrivals;
  }
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
    return launch(attn_tc_kernel, dim3(pl.splits, pl.n_tiles, p.batch * p.hkv), dim3(kThreads),
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
