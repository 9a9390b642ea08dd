// Target LM head with the acceptance's row statistics in its epilogue (LTD
// section 3.2, "Draft Tree Verification": one target forward over the
// verified tokens, whose last layer maps each hidden state to vocabulary
// logits; acceptance then needs each row's max, log-sum-exp and argmax).
//
// logits[r][v] = sum_k hidden[r][k] weight[v][k], bf16 inputs, fp32
// accumulation, on the tensor cores with the operands swapped: a CTA
// computes D = W_tile H^T for 128-row vocabulary tiles of the weight (the M
// side of tcgen05.mma) against every hidden row (the N side, up to 256), so
// the weight -- the bytes that bound this step -- streams through once.
//   warp 0      TMA: per 64-element k-block, the weight tile's 128 rows and
//               all hidden rows into a ring of stages (128-byte swizzle);
//   warp 1      tcgen05.mma into one of two tensor-memory accumulators, so
//               a tile's epilogue overlaps the next tile's MMAs;
//   warps 4-7   epilogue, one thread per vocabulary row (= TMEM lane): per
//               hidden row, the tile's (max, argmax) by a warp max of
//               (logit, token) keys and its sum of exp(x - max), merged
//               over the warps and into the CTA's running statistics;
//               optionally the logits themselves (bf16).
// A second kernel merges the CTAs' statistics per row, a warp per row (the
// launch boundary orders it after every CTA's writes), and writes max, LSE,
// argmax.
#include "ltd_common.cuh"
#include "ltd_internal.h"
#include "tc_util.cuh"

namespace ltd {

namespace {

constexpr int kVT = 128;                  // vocabulary rows per tile (MMA M, TMEM lanes)
constexpr int kKB = 64;                   // hidden elements per k-block (one 128-byte atom)
constexpr int kThreads = 256;             // TMA, MMA, 2 idle, 4 epilogue warps
constexpr uint32_t kTileA = kVT * 128;    // bytes of one weight k-block
constexpr uint32_t kStageMax = 8;
constexpr uint32_t kSmemBudget = 200 * 1024;
constexpr int kMaxGrid = 256;             // the merge kernel takes up to 256 CTAs' statistics

struct LmArgs {
  int32_t rows, n_pad, hidden, kblocks, tiles, stages;  // n_pad: rows rounded up to 32
  int64_t vocab;
  __nv_bfloat16* logits;  // [rows][vocab] or null
  float* part;            // [grid][n_pad] x (m, s) as float2
  unsigned long long* part_key;  // [grid][n_pad] argmax keys
  uint32_t* err;
};

// statistics of a set of logits: max m, sum of exp(x - m), argmax key
struct Stat {
  float m, s;
  unsigned long long key;
};
__device__ __forceinline__ void stat_merge(Stat& a, const Stat& b) {
  if (b.m == -CUDART_INF_F) return;
  if (a.m == -CUDART_INF_F) {
    a = b;
    return;
  }
  const float mm = fmaxf(a.m, b.m);
  a.s = a.s * __expf(a.m - mm) + b.s * __expf(b.m - mm);
  a.m = mm;
  a.key = b.key > a.key ? b.key : a.key;
}

__global__ void __launch_bounds__(kThreads, 1)
    lm_head_kernel(const __grid_constant__ CUtensorMap tw, const __grid_constant__ CUtensorMap th,
                   const LmArgs a) {
  extern __shared__ uint8_t smem_raw[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t raw = tc::smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  const uint32_t tileB = static_cast<uint32_t>(a.n_pad) * 128u;  // bytes of one hidden k-block
  const uint32_t stage_bytes = kTileA + tileB;
  const int S = a.stages;
  // layout: stages | warp partials [4][n_pad] Stat | running [n_pad] Stat | barriers | holder
  const uint32_t off_part = static_cast<uint32_t>(S) * stage_bytes;
  const uint32_t off_run = off_part + 4u * a.n_pad * sizeof(Stat);
  const uint32_t off_bar = off_run + static_cast<uint32_t>(a.n_pad) * sizeof(Stat);
  Stat* wpart = reinterpret_cast<Stat*>(gbase + off_part);
  Stat* run = reinterpret_cast<Stat*>(gbase + off_run);
  auto full = [&](int i) { return base + off_bar + 8u * i; };
  auto empty = [&](int i) { return base + off_bar + 8u * (kStageMax + i); };
  auto accfull = [&](int i) { return base + off_bar + 8u * (2 * kStageMax + i); };
  auto accempty = [&](int i) { return base + off_bar + 8u * (2 * kStageMax + 2 + i); };
  uint32_t* holder = reinterpret_cast<uint32_t*>(gbase + off_bar + 8u * (2 * kStageMax + 4));
  // two accumulators of n_pad columns, each at a power-of-two column offset
  const uint32_t tmem_cols = a.n_pad * 2 <= 64 ? 64u : (a.n_pad * 2 <= 128 ? 128u : (a.n_pad * 2 <= 256 ? 256u : 512u));
  const uint32_t bufcols = tmem_cols / 2;

  if (tid == 0) {
    tc::tma_prefetch(&tw);
    tc::tma_prefetch(&th);
    for (int i = 0; i < S; ++i) {
      tc::mbar_init(full(i), 1);
      tc::mbar_init(empty(i), 1);
    }
    for (int i = 0; i < 2; ++i) {
      tc::mbar_init(accfull(i), 1);
      tc::mbar_init(accempty(i), 1);
    }
    tc::mbar_init_fence();
  }
  if (warp == 1) {
    tc::tmem_alloc(tc::smem_u32(holder), tmem_cols);
    tc::tmem_relinquish();
  }
  for (int c = tid; c < a.n_pad; c += kThreads) run[c] = Stat{-CUDART_INF_F, 0.f, 0ull};
  grid_wait();
  trigger_dependents();
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = holder[0];
  const int G = gridDim.x;
  const int my_tiles = a.tiles > static_cast<int>(blockIdx.x) ? (a.tiles - 1 - blockIdx.x) / G + 1 : 0;
  bool ok = true;

  if (warp == 0) {
    // --------------------------------------------------------- producer
    if (lane == 0) {
      int it = 0;
      for (int t = 0; t < my_tiles && ok; ++t) {
        const int tile = blockIdx.x + t * G;
        for (int kb = 0; kb < a.kblocks && ok; ++kb, ++it) {
          const int st = it % S, use = it / S;
          if (it >= S) ok = tc::mbar_wait(empty(st), (use - 1) & 1);
          if (!ok) break;
          const uint32_t dst = base + st * stage_bytes;
          tc::mbar_expect_tx(full(st), stage_bytes);
          tc::tma_load_3d(dst, &tw, full(st), kb * kKB, tile * kVT, 0);
          tc::tma_load_3d(dst + kTileA, &th, full(st), kb * kKB, 0, 0);
        }
      }
      // every load issued lands before the CTA leaves (one per stage at most
      // is outstanding: a stage is reloaded only after its MMAs completed)
      const int issued = it;
      for (int st = 0; st < S && st < issued; ++st) {
        const int last = st + ((issued - 1 - st) / S) * S;  // last use of this stage
        tc::mbar_wait(full(st), (last / S) & 1);
      }
      if (!ok) flag_error(a.err, LTD_DEVERR_TIMEOUT);
    }
  } else if (warp == 1) {
    // -------------------------------------------------------------- MMA
    if (lane == 0 && my_tiles > 0) {
      const uint32_t idesc = tc::idesc_bf16(kVT, a.n_pad, false);
      const uint64_t da0 = tc::sdesc_sw128(base, 16, 1024);
      const uint64_t db0 = tc::sdesc_sw128(base + kTileA, 16, 1024);
      int it = 0;
      for (int t = 0; t < my_tiles && ok; ++t) {
        const int buf = t & 1;
        if (t >= 2) ok = tc::mbar_wait(accempty(buf), ((t >> 1) - 1) & 1);
        if (!ok) break;
        tc::fence_after_sync();
        const uint32_t d = tmem + buf * bufcols;
        for (int kb = 0; kb < a.kblocks && ok; ++kb, ++it) {
          const int st = it % S, use = it / S;
          ok = tc::mbar_wait(full(st), use & 1);
          if (!ok) break;
          tc::fence_after_sync();
          const uint64_t so = static_cast<uint64_t>((st * stage_bytes) >> 4);
#pragma unroll
          for (int ks = 0; ks < 4; ++ks)
            tc::mma_bf16(d, da0 + so + ks * 2, db0 + so + ks * 2, idesc, (kb | ks) ? 1u : 0u);
          tc::mma_commit(empty(st));
        }
        if (ok) tc::mma_commit(accfull(buf));
      }
      if (!ok) flag_error(a.err, LTD_DEVERR_TIMEOUT);
    }
  } else if (warp >= 4) {
    // --------------------------------------------------------- epilogue
    const int e = tid - 128;  // vocabulary row of the tile = TMEM lane
    const int wq = warp - 4;
    const uint32_t lane_off = (32u * wq) << 16;
    for (int t = 0; t < my_tiles && ok; ++t) {
      const int tile = blockIdx.x + t * G;
      const int buf = t & 1;
      // one decision for the four warps, which meet at named barriers below
      ok = tc::bar_red_and(1, 128, tc::mbar_wait(accfull(buf), (t >> 1) & 1));
      if (!ok) break;
      tc::fence_after_sync();
      const int64_t v = static_cast<int64_t>(tile) * kVT + e;
      const bool valid = v < a.vocab;
      for (int c0 = 0; c0 < a.n_pad; c0 += 32) {
        tc::Frag32 f;
        tc::tmem_ld32_sync(tmem + buf * bufcols + c0 + lane_off, f);
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          const int r = c0 + j;
          const float x = valid ? __uint_as_float(f.r[j]) : -CUDART_INF_F;
          if (a.logits != nullptr && valid && r < a.rows)
            a.logits[static_cast<int64_t>(r) * a.vocab + v] = __float2bfloat16_rn(x);
          unsigned long long k = valid ? make_key(x, static_cast<uint32_t>(v)) : 0ull;
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) {
            const unsigned long long ok2 = __shfl_xor_sync(0xFFFFFFFFu, k, o);
            k = ok2 > k ? ok2 : k;
          }
          const float m = k != 0ull ? key_value(k) : -CUDART_INF_F;
          float s = (valid && m != -CUDART_INF_F) ? __expf(x - m) : 0.f;
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xFFFFFFFFu, s, o);
          if (lane == 0) wpart[wq * a.n_pad + r] = Stat{m, s, k};
        }
      }
      // this tile's accumulator may be overwritten once every epilogue
      // thread has read it
      tc::fence_before_sync();
      asm volatile("bar.sync 1, 128;" ::: "memory");
      if (e == 0) tc::mbar_arrive(accempty(buf));
      for (int r = e; r < a.rows; r += 128) {
        Stat acc = run[r];
#pragma unroll
        for (int w = 0; w < 4; ++w) stat_merge(acc, wpart[w * a.n_pad + r]);
        run[r] = acc;
      }
      asm volatile("bar.sync 1, 128;" ::: "memory");  // partials read before the next tile
    }
    if (!ok && e == 0) flag_error(a.err, LTD_DEVERR_TIMEOUT);
    // this CTA's statistics for the merge kernel
    for (int r = e; r < a.n_pad; r += 128) {
      const Stat st = run[r];
      reinterpret_cast<float2*>(a.part)[static_cast<int64_t>(blockIdx.x) * a.n_pad + r] =
          make_float2(st.m, st.s);
      a.part_key[static_cast<int64_t>(blockIdx.x) * a.n_pad + r] = st.key;
    }
  }
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, tmem_cols);
  }
}

// A warp per row: lane l merges the statistics of CTAs l, l + 32, ... (its
// loads issued together), then the lanes merge pairwise in a fixed tree, so
// the result does not depend on timing.  The launch boundary orders this
// after every write of the first kernel.
constexpr int kMergeWarps = 8;
__global__ void __launch_bounds__(kMergeWarps * 32)
    lm_head_merge_kernel(const float* part, const unsigned long long* part_key, int grid,
                         int n_pad, int rows, float* row_max, float* row_lse, int32_t* row_argmax) {
  grid_wait();
  trigger_dependents();
  const int lane = threadIdx.x & 31;
  const int r = blockIdx.x * kMergeWarps + (threadIdx.x >> 5);
  if (r >= rows) return;
  constexpr int kPer = kMaxGrid / 32;
  float2 ms[kPer];
  unsigned long long ky[kPer];
#pragma unroll
  for (int i = 0; i < kPer; ++i) {
    const int c = lane + 32 * i;
    ms[i] = c < grid ? reinterpret_cast<const float2*>(part)[static_cast<int64_t>(c) * n_pad + r]
                     : make_float2(-CUDART_INF_F, 0.f);
    ky[i] = c < grid ? part_key[static_cast<int64_t>(c) * n_pad + r] : 0ull;
  }
  Stat acc{-CUDART_INF_F, 0.f, 0ull};
#pragma unroll
  for (int i = 0; i < kPer; ++i) stat_merge(acc, Stat{ms[i].x, ms[i].y, ky[i]});
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    Stat other;
    other.m = __shfl_xor_sync(0xFFFFFFFFu, acc.m, o);
    other.s = __shfl_xor_sync(0xFFFFFFFFu, acc.s, o);
    other.key = __shfl_xor_sync(0xFFFFFFFFu, acc.key, o);
    // both lanes of a pair merge the same two values in the same order
    Stat lo = (lane & o) ? other : acc, hi = (lane & o) ? acc : other;
    stat_merge(lo, hi);
    acc = lo;
  }
  if (lane == 0) {
    row_max[r] = acc.m;
    row_lse[r] = acc.m + logf(acc.s);
    row_argmax[r] = static_cast<int32_t>(key_index(acc.key));
  }
}

}  // namespace

size_t lm_head_workspace(int32_t rows, int64_t vocab) {
  const int n_pad = (rows + 31) / 32 * 32;
  const int64_t tiles = (vocab + kVT - 1) / kVT;
  int grid = device_sm_count();
  if (grid > kMaxGrid) grid = kMaxGrid;
  if (tiles < grid) grid = static_cast<int>(tiles);
  return static_cast<size_t>(grid) * n_pad * (sizeof(float2) + sizeof(unsigned long long)) + 256;
}

cudaError_t launch_lm_head(const LmHeadParams& p, cudaStream_t s) {
  LmArgs a{};
  a.rows = p.rows;
  a.n_pad = (p.rows + 31) / 32 * 32;  // whole 32-column epilogue chunks
  a.hidden = p.hidden;
  a.kblocks = p.hidden / kKB;
  a.vocab = p.vocab;
  a.tiles = static_cast<int32_t>((p.vocab + kVT - 1) / kVT);
  const uint32_t stage_bytes = kTileA + static_cast<uint32_t>(a.n_pad) * 128u;
  a.stages = static_cast<int32_t>(kSmemBudget / stage_bytes);
  if (a.stages > static_cast<int32_t>(kStageMax)) a.stages = kStageMax;
  if (a.stages < 2) return cudaErrorInvalidValue;
  int grid = device_sm_count();
  if (grid > kMaxGrid) grid = kMaxGrid;
  if (a.tiles < grid) grid = a.tiles;
  const size_t need = static_cast<size_t>(grid) * a.n_pad * (sizeof(float2) + sizeof(unsigned long long));
  if (p.ws == nullptr || p.ws_bytes < need) return cudaErrorInvalidValue;
  a.logits = static_cast<__nv_bfloat16*>(p.logits);
  a.part = static_cast<float*>(p.ws);
  a.part_key = reinterpret_cast<unsigned long long*>(static_cast<uint8_t*>(p.ws) +
                                                     static_cast<size_t>(grid) * a.n_pad * sizeof(float2));
  a.err = p.err;
  CUtensorMap tw, th;
  const uint64_t row = static_cast<uint64_t>(p.hidden) * 2;
  if (!encode_tmap_bf16_3d(&tw, p.weight, p.hidden, p.vocab, 1, row, row * p.vocab, kKB, kVT, 1) ||
      !encode_tmap_bf16_3d(&th, p.hidden_states, p.hidden, p.rows, 1, row, row * p.rows, kKB, a.n_pad, 1))
    return cudaErrorInvalidValue;
  const size_t smem = static_cast<size_t>(a.stages) * stage_bytes +
                      static_cast<size_t>(5) * a.n_pad * sizeof(Stat) + 8 * (2 * kStageMax + 4) + 16 + 1024;
  cudaError_t e = cudaFuncSetAttribute(lm_head_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  e = launch(lm_head_kernel, dim3(grid), dim3(kThreads), smem, s, nullptr, 0, tw, th, a);
  if (e != cudaSuccess) return e;
  return launch(lm_head_merge_kernel, dim3((a.rows + kMergeWarps - 1) / kMergeWarps),
                dim3(kMergeWarps * 32), 0, s, nullptr, 0,
                static_cast<const float*>(a.part), static_cast<const unsigned long long*>(a.part_key),
                grid, a.n_pad, a.rows, p.row_max, p.row_lse, p.row_argmax);
}

}  // namespace ltd
