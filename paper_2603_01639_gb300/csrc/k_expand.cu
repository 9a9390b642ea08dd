// Draft tree generation (LTD section 3.2, "Draft Tree Generation").
//
// One launch builds one level for every active sequence: F = 1 row (the
// root's) at level 1, F = k rows (one per frontier node) afterwards.  Every
// row is cut into items of 16 KB (8192 bf16 or 4096 fp32 entries); a
// cooperative grid of at most two CTAs per SM takes contiguous runs of
// items, each staged into shared memory by a bulk copy (three buffers in
// flight per CTA, each with its mbarrier).
//
// Per item (producer): each of the 512 threads takes two 16-byte vectors,
// their max and their sum of exp.  The k-th largest of the 32 half-warp
// maxima, T, bounds the item's k-th largest logit from below (k half-warps
// hold an entry >= T), so only the entries >= T -- typically a few dozen --
// can be among the item's top-k; they go to a shared list and each finds its
// rank by counting the larger ones.  The item's record -- its top-k keys
// (logit desc, token asc) and its (max, sum of exp) -- goes to the tree's
// scratch area, every 64-bit word tagged with the level.  Items whose list
// overflows (huge tie sets) are ranked exactly by warp top-k lists.
//
// Per sequence (consumer): the CTA that holds the sequence's last item,
// after its own items, waits (bounded) until every word of the sequence's
// records carries the level's tag, copies them to shared memory and merges
// them, one warp per row: the row's threshold is the k-th largest of its
// items' leading keys (at least k keys reach it, typically few more), the
// keys that reach it are ranked by counting, and the row's k children get
// cum = cum(parent) + x - logsumexp(row) (fp32).  The new frontier, the k
// best of the F k children by (cum desc, node id asc), is ranked the same
// way.  ltd_tree_reset zeroes the scratch area, so no record of an earlier
// cycle carries a live tag and a record of an earlier level carries another.
//
// The kernel's code is kept small: its consumer runs once per launch on one
// SM, where instructions that are not cached cost about three cycles each.
// Shapes whose records exceed the consumer's buffer use a second
// instantiation that merges the rows' lists in warps.
#include "ltd_common.cuh"
#include "ltd_internal.h"
#include "tc_util.cuh"

#include <mutex>

namespace ltd {

namespace {

constexpr int kNT = 512;
constexpr int kNW = kNT / kWarp;
constexpr int kStages = 3;        // item buffers in flight per CTA
constexpr int kItemBytes = 16384;
constexpr int kCand = 512;        // producer: candidate list capacity per item
constexpr int kRecBuf = 2560;     // consumer: a sequence's record words in shared memory
constexpr int kRowCand = 48;      // consumer: candidates kept per row
constexpr int kBatch = 8;         // large-shape consumer: item lists a warp loads per pass
constexpr int kTagShift = 20;     // word: value bits << 32 | tag << 20 | (2^20 - 1 - token)
constexpr uint32_t kIdxMask = (1u << kTagShift) - 1u;
static_assert(kExpandMaxVocab <= (int64_t(1) << kTagShift), "token ids fit the word's index field");
static_assert(kItemBytes == kNT * 2 * 16, "an item is two 16-byte vectors per thread");

// Optional phase timestamps for performance work (off in normal builds).
#ifdef LTD_TRACE
__device__ unsigned long long g_expand_trace[4096][8];
#define TRACE(slot)                                                   \
  do {                                                                \
    if (threadIdx.x == 0 && blockIdx.x < 4096)                        \
      g_expand_trace[blockIdx.x][slot] = tc::globaltimer();           \
  } while (0)
#else
#define TRACE(slot) \
  do {              \
  } while (0)
#endif

// Starts a cycle: the root of every tree, and the scratch area zeroed (16
// bytes per thread over the whole grid).
__global__ void tree_reset_kernel(ltd_tree t, const int32_t* __restrict__ roots, uint4* scratch,
                                  int64_t scratch_vecs) {
  grid_wait();
  trigger_dependents();
  const int64_t g = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  for (int64_t i = g; i < scratch_vecs; i += static_cast<int64_t>(gridDim.x) * blockDim.x)
    scratch[i] = make_uint4(0u, 0u, 0u, 0u);
  if (g >= t.batch) return;
  const int b = static_cast<int>(g);
  const int64_t nb = static_cast<int64_t>(b) * t.max_nodes;
  t.token[nb] = roots[b];
  t.parent[nb] = -1;
  t.depth[nb] = 0;
  t.cum_logprob[nb] = 0.f;
  t.xrow[nb] = -1;
  t.xlse[nb] = 0.f;
  t.n_nodes[b] = 1;
  t.n_levels[b] = 0;
  for (int i = 0; i < t.k; ++i) t.frontier[b * t.k + i] = (i == 0) ? 0 : -1;
}

// ------------------------------------------------------ tagged record words
// Every word: the value's bits above, the tag and the complemented token
// below.  Keys use the value's order bits, so a larger word is a larger
// value, then a lower token (as make_key); an empty slot has value bits 0,
// below every real key.  Statistics use the float's own bits.
__device__ __forceinline__ uint64_t tagged_key(float v, uint32_t token, uint32_t tag) {
  return (static_cast<uint64_t>(float_order_bits(v)) << 32) |
         static_cast<uint64_t>((tag << kTagShift) | (kIdxMask - token));
}
__device__ __forceinline__ uint64_t tagged_empty(uint32_t tag) {
  return static_cast<uint64_t>(tag << kTagShift);
}
__device__ __forceinline__ uint64_t tagged_stat(float v, uint32_t tag) {
  return (static_cast<uint64_t>(__float_as_uint(v)) << 32) | static_cast<uint64_t>(tag << kTagShift);
}
__device__ __forceinline__ uint32_t word_tag(uint64_t w) {
  return static_cast<uint32_t>(w) >> kTagShift;
}
__device__ __forceinline__ uint32_t tagged_token(uint64_t w) {
  return kIdxMask - (static_cast<uint32_t>(w) & kIdxMask);
}
__device__ __forceinline__ float key_float(uint64_t w) {
  return order_bits_float(static_cast<uint32_t>(w >> 32));
}
__device__ __forceinline__ float stat_float(uint64_t w) {
  return __uint_as_float(static_cast<uint32_t>(w >> 32));
}

__device__ __forceinline__ void st_relaxed(uint64_t* p, uint64_t v) {
  asm volatile("st.relaxed.gpu.global.b64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}
__device__ __forceinline__ uint64_t ld_relaxed(const uint64_t* p) {
  uint64_t v;
  asm volatile("ld.relaxed.gpu.global.b64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}
// A 32-bit load through L2 that the compiler issues where it is written
// (volatile asm), not next to its first use.
__device__ __forceinline__ int32_t ld_cg_early(const int32_t* p) {
  int32_t v;
  asm volatile("ld.global.cg.b32 %0, [%1];" : "=r"(v) : "l"(p));
  return v;
}

// ------------------------------------------------------------ shared memory
struct ExpandHead {
  uint64_t bar[kStages];  // item buffers' mbarriers
  float gmax[2 * kNW];    // half-warp maxima of the current item
  float wsum[kNW];        // the warps' sums of exp(x - item max)
  float thr, cmax;        // the current item's threshold and max
  int n_cand[2];          // candidate counts, by item parity
  int stage_on[kStages];  // whether the buffer's item was loaded
  int load_fail;          // an item buffer's wait ran out: no more records
  int fail;               // consumer: a wait ran out
};
struct ProducerShared {
  uint4 ring[kStages][kItemBytes / 16];
  uint64_t cand[kCand];
  uint64_t lists[kNW * kWarp];  // exact fallback's warp lists
};
struct ConsumerShared {
  uint64_t rec[kRecBuf];                  // the sequence's records, [row][item][k + 2]
  uint64_t cand[LTD_MAX_K][kRowCand];     // each row's candidates
  uint64_t child[LTD_MAX_K * LTD_MAX_K];  // [row][rank] child keys (cum, node id)
  uint64_t top[LTD_MAX_K * LTD_MAX_K];    // [row][rank] each row's top keys
  uint64_t vals[LTD_MAX_K * kWarp];       // [row] leading keys (scratch)
  unsigned long long trow[LTD_MAX_K];     // row thresholds (general path)
  float lse[LTD_MAX_K];
  float cum_p[LTD_MAX_K];
  int parent[LTD_MAX_K];
};
struct alignas(128) ExpandShared {
  ExpandHead h;
  alignas(128) union {
    ProducerShared pr;
    ConsumerShared co;
  } u;
};

// Where an item lives: sequence b, row slot f, chunk c of the row.  Items
// are numbered row-major over (b, f, c) and visited in order.
struct Item {
  int b, f, c;
};
__device__ __forceinline__ Item item_at(const ExpandParams& p, int it) {
  Item q;
  q.c = it % p.chunks;
  const int bf = it / p.chunks;
  q.f = bf % p.F;
  q.b = bf / p.F;
  return q;
}
__device__ __forceinline__ void advance(const ExpandParams& p, Item& q) {
  if (++q.c == p.chunks) {
    q.c = 0;
    if (++q.f == p.F) {
      q.f = 0;
      ++q.b;
    }
  }
}
__device__ __forceinline__ int64_t draft_row(const ExpandParams& p, int f) {
  return (p.level == 1) ? 0 : 1 + static_cast<int64_t>(p.level - 2) * p.k + f;
}
// A sequence's records: F rows x chunks items x (k + 2) words, contiguous.
__device__ __forceinline__ uint64_t* seq_records(const ExpandParams& p, int b) {
  return p.rec + static_cast<int64_t>(b) * p.F * p.chunks * (p.k + 2);
}
__device__ __forceinline__ bool seq_active(const ExpandParams& p, int b) {
  return p.active == nullptr || __ldcg(p.active + b) != 0;
}

// ---------------------------------------------------------------- producer
// Thread 0: item q's bytes into ring buffer s (one bulk copy completing on
// the buffer's mbarrier), or, for an item of an inactive sequence, a plain
// arrival so the buffer's phases stay in step.
template <typename T>
__device__ __forceinline__ void issue_item(const ExpandParams& p, ExpandShared& sh, int s, const Item& q) {
  const uint32_t bar = tc::smem_u32(&sh.h.bar[s]);
  const bool on = seq_active(p, q.b);
  sh.h.stage_on[s] = on ? 1 : 0;
  if (!on) {
    tc::mbar_arrive(bar);
    return;
  }
  const int lo = q.c * p.item_elems;
  const int n = min(p.item_elems, static_cast<int>(p.vocab) - lo);
  const T* src = reinterpret_cast<const T*>(p.rows) +
                 (static_cast<int64_t>(q.b) * p.rows_per_seq + draft_row(p, q.f)) * p.vocab + lo;
  const uint32_t bytes = static_cast<uint32_t>(n) * static_cast<uint32_t>(sizeof(T));  // multiple of 16
  tc::mbar_expect_tx(bar, bytes);
  tc::bulk_g2s(tc::smem_u32(&sh.u.pr.ring[s][0]), src, bytes, bar);
}

// Exact top-k of an item whose candidate list overflowed (huge tie sets):
// every entry is offered to its warp's list, the lists are merged, and
// threads tid < k store the result.  Out of line: it is rarely run.
template <typename T>
__device__ __noinline__ void exact_item_topk(const ExpandParams& p, ExpandShared& sh, const T* item, int lo,
                                             int n_here, uint32_t tag, uint64_t* rec, bool write) {
  constexpr int VEC = 16 / sizeof(T);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  WarpTopK wt;
  wt.init();
#pragma unroll 1
  for (int e = 0; e < 2 * VEC; ++e) {
    const int off = ((e / VEC) * kNT + tid) * VEC + e % VEC;
    wt.offer(off < n_here ? tagged_key(to_f(item[off]), static_cast<uint32_t>(lo + off), tag) : 0ull, p.k);
  }
  sh.u.pr.lists[warp * kWarp + lane] = wt.v;
#pragma unroll 1
  for (int step = 1; step < kNW; step <<= 1) {
    __syncthreads();
    if ((warp % (2 * step)) == 0 && warp + step < kNW) {
      const uint64_t m = warp_merge_desc(sh.u.pr.lists[warp * kWarp + lane],
                                         sh.u.pr.lists[(warp + step) * kWarp + lane]);
      __syncwarp();
      sh.u.pr.lists[warp * kWarp + lane] = m;
    }
  }
  __syncthreads();
  if (tid < p.k && write) st_relaxed(rec + tid, sh.u.pr.lists[tid]);
}

// One item: its top-k keys and (max, sum of exp) into its record.  Every
// thread of the CTA calls it (block barriers inside); `parity` alternates
// between consecutive calls.  `item` is the item's buffer.
template <typename T>
__device__ __forceinline__ void produce_item(const ExpandParams& p, ExpandShared& sh, const Item& q,
                                             const T* item, bool write, int parity) {
  constexpr int VEC = 16 / sizeof(T);
  constexpr int U = 2;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int k = p.k;
  const uint32_t tag = static_cast<uint32_t>(p.level);
  const int lo = q.c * p.item_elems;  // vocab <= 2^20: 32-bit offsets
  const int n_here = min(p.item_elems, static_cast<int>(p.vocab) - lo);
  // ---- the thread's two vectors; a vector past the row's end (only a
  // row's last item is partial, and it ends on a vector boundary) reads as
  // -inf.  Then the thread's max and sum of exp.
  uint4 raw[U];
#pragma unroll
  for (int u = 0; u < U; ++u) {
    raw[u] = reinterpret_cast<const uint4*>(item)[u * kNT + tid];
    if ((u * kNT + tid) * VEC >= n_here)
      raw[u] = (sizeof(T) == 4) ? make_uint4(0xFF800000u, 0xFF800000u, 0xFF800000u, 0xFF800000u)
                                : make_uint4(0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u);
  }
  float tmax = -CUDART_INF_F, tsum = 0.f;
#pragma unroll
  for (int u = 0; u < U; ++u)
#pragma unroll
    for (int j = 0; j < VEC; ++j) tmax = fmaxf(tmax, elem<T>(raw[u], j));
  if (tmax > -CUDART_INF_F) {
#pragma unroll
    for (int u = 0; u < U; ++u)
#pragma unroll
      for (int j = 0; j < VEC; ++j) tsum += __expf(elem<T>(raw[u], j) - tmax);
  }
  // ---- T = k-th largest of the 32 half-warp maxima (k half-warps hold an
  // entry >= T, so the item's top-k are >= T), the item's max = the largest;
  // warp 0 ranks the maxima by counting (ties to the lower slot)
  float hm = tmax;
#pragma unroll
  for (int o = 8; o > 0; o >>= 1) hm = fmaxf(hm, __shfl_xor_sync(0xFFFFFFFFu, hm, o));
  if ((lane & 15) == 0) sh.h.gmax[warp * 2 + (lane >> 4)] = hm;
  __syncthreads();
  if (warp == 0) {
    const float mine = sh.h.gmax[lane];
    int rank = 0;
#pragma unroll 8
    for (int j = 0; j < 32; ++j) {
      const float o = sh.h.gmax[j];
      rank += (o > mine || (o == mine && j < lane)) ? 1 : 0;
    }
    if (rank == k - 1) sh.h.thr = mine;
    if (rank == 0) sh.h.cmax = mine;
    if (lane == 0) sh.h.n_cand[parity ^ 1] = 0;  // last read before the barrier above
  }
  __syncthreads();
  const float thr = sh.h.thr, cmax = sh.h.cmax;
  // ---- the candidates >= T (the thread's bits), one reservation each
  uint32_t cm = 0u;
  if (tmax >= thr) {
#pragma unroll
    for (int u = 0; u < U; ++u)
      if ((u * kNT + tid) * VEC < n_here)  // (whole vectors lie inside or past the row)
#pragma unroll
        for (int j = 0; j < VEC; ++j)
          if (elem<T>(raw[u], j) >= thr) cm |= 1u << (u * VEC + j);
  }
  if (cm != 0u) {
    int slot = atomicAdd(&sh.h.n_cand[parity], __popc(cm));
#pragma unroll 1
    while (cm != 0u) {
      const int e = __ffs(cm) - 1;
      cm &= cm - 1u;
      const int off = ((e / VEC) * kNT + tid) * VEC + e % VEC;
      if (slot < kCand) sh.u.pr.cand[slot] = tagged_key(to_f(item[off]), static_cast<uint32_t>(lo + off), tag);
      ++slot;
    }
  }
  {
    float e = (tmax > -CUDART_INF_F) ? tsum * __expf(tmax - cmax) : 0.f;
    e = warp_sum_f(e);
    if (lane == 0) sh.h.wsum[warp] = e;
  }
  __syncthreads();
  const int nc = sh.h.n_cand[parity];
  write = write && sh.h.load_fail == 0;
  uint64_t* rec = seq_records(p, q.b) + (static_cast<int64_t>(q.f) * p.chunks + q.c) * (k + 2);
  if (nc <= kCand) {
    // each candidate's rank = the number of larger ones (keys are unique)
    if (tid < nc) {
      const uint64_t key = sh.u.pr.cand[tid];
      int r = 0;
#pragma unroll 8
      for (int i = 0; i < nc; ++i) r += (sh.u.pr.cand[i] > key) ? 1 : 0;
      if (write && r < k) st_relaxed(rec + r, key);
    }
    if (tid >= nc && tid < k && write) st_relaxed(rec + tid, tagged_empty(tag));  // fewer than k entries
  } else {
    exact_item_topk<T>(p, sh, item, lo, n_here, tag, rec, write);
  }
  if (warp == kNW - 1 && write) {
    float s = lane < kNW ? sh.h.wsum[lane] : 0.f;
    s = warp_sum_f(s);
    if (lane == 0) {
      st_relaxed(rec + k, tagged_stat(cmax, tag));
      st_relaxed(rec + k + 1, tagged_stat(s, tag));
    }
  }
}

// ---------------------------------------------------------------- consumer
// What the merging CTA fetches for its sequence while its items load: the
// sequence (-1: none), its active flag and level word, and for thread f < F
// the frontier node of rank f (row f's parent) and its cum.
struct ConsumerPrefetch {
  int b;
  int act, lev;
  int parent;
  float cum;
};

// Thread f < F: row f's parent and its cum into shared memory, from the
// prefetch when it is this sequence's.
__device__ __forceinline__ void load_parent(const ExpandParams& p, const ConsumerPrefetch& pf, int b,
                                            int64_t nb, ConsumerShared& co) {
  const int f = threadIdx.x;
  int parent = 0;
  float cum = 0.f;
  if (p.level > 1) {
    if (pf.b == b) {
      parent = pf.parent;
      cum = pf.cum;
    } else {
      parent = __ldcg(&p.frontier[b * p.k + f]);
      cum = __ldcg(&p.cum[nb + parent]);
    }
  }
  co.parent[f] = parent;
  co.cum_p[f] = cum;
}

// Child of rank r of row f, from its key (value, token).
__device__ __forceinline__ void write_child(const ExpandParams& p, ConsumerShared& co, int64_t nb,
                                            int base, int f, int r, uint64_t key) {
  const int id = base + f * p.k + r;
  const float cum = co.cum_p[f] + (key_float(key) - co.lse[f]);
  const int64_t g = nb + id;
  p.token[g] = static_cast<int32_t>(tagged_token(key));
  p.parent[g] = co.parent[f];
  p.depth[g] = p.level;
  p.cum[g] = cum;
  p.xrow[g] = -1;
  p.xlse[g] = 0.f;
  co.child[f * p.k + r] = make_key(cum, static_cast<uint32_t>(id));
}

// One warp, row f's log-sum-exp from its items' (max, sum of exp): lane
// 0's value for the whole row, so tied children get bit-identical cums.
__device__ __forceinline__ float row_lse(const uint64_t* row, int C, int rw, int k) {
  const int lane = threadIdx.x & 31;
  float M = -CUDART_INF_F;
#pragma unroll 1
  for (int c = lane; c < C; c += kWarp) M = fmaxf(M, stat_float(row[c * rw + k]));
  M = warp_max_f(M);
  float S = 0.f;
  if (M > -CUDART_INF_F)
#pragma unroll 1
    for (int c = lane; c < C; c += kWarp) S += stat_float(row[c * rw + k + 1]) * __expf(stat_float(row[c * rw + k]) - M);
  S = warp_sum_f(S);
  return __shfl_sync(0xFFFFFFFFu, M + __logf(S), 0);
}

// One warp: the k largest keys of L sorted lists (list i at lists + i
// stride, k keys each, descending; keys unique except empty ones, which
// never make the cut), in rank order into top[0..k).  With J > 0 (from the
// host: L J <= 32 and L J >= k) the threshold T is the k-th largest of the
// lists' first J keys (lane a holds key a / L of list a mod L): at least k
// keys reach it, so the top k do, and typically little more than k do;
// those (each list's first few, as it is sorted) are compacted into cand and
// ranked by counting the larger ones.  With J = 0, or more candidates than
// cand holds, every key is ranked against all keys (slow, rare).  vals: 32
// words of scratch.
__device__ __forceinline__ void warp_topk_lists(const uint64_t* lists, int L, int stride, int k, int J,
                                                uint64_t* vals, uint64_t* cand, uint64_t* top) {
  const int lane = threadIdx.x & 31;
  uint64_t T = 0ull;  // (0: every key a candidate)
  int total = kRowCand + 1;
  if (J > 0) {
    // ---- threshold
    const int LJ = L * J;
    const int ja = __float2int_rd(static_cast<float>(lane) * __frcp_rn(static_cast<float>(L)) + 1e-4f);
    const uint64_t mine = lane < LJ ? lists[(lane - ja * L) * stride + ja] : 0ull;
    vals[lane] = mine;
    __syncwarp();
    int r = 0;
#pragma unroll 4
    for (int j = 0; j < LJ; ++j) r += (vals[j] > mine) ? 1 : 0;
    const uint32_t hit = __ballot_sync(0xFFFFFFFFu, lane < LJ && r == k - 1);  // (none: tied empties)
    if (hit != 0u) T = __shfl_sync(0xFFFFFFFFu, mine, __ffs(hit) - 1);
    // ---- candidates: list `lane`'s keys >= T (a prefix)
    int n = 0;
    if (lane < L)
      while (n < k && lists[lane * stride + n] >= T) ++n;
    int incl = n;
#pragma unroll
    for (int o = 1; o < kWarp; o <<= 1) {
      const int y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
      if (lane >= o) incl += y;
    }
    total = __shfl_sync(0xFFFFFFFFu, incl, kWarp - 1);
    if (total <= kRowCand)
      for (int j = 0; j < n; ++j) cand[incl - n + j] = lists[lane * stride + j];
  }
  __syncwarp();
  if (total <= kRowCand) {
    for (int i = lane; i < total; i += kWarp) {
      const uint64_t key = cand[i];
      int r = 0;
#pragma unroll 4
      for (int j = 0; j < total; ++j) r += (cand[j] > key) ? 1 : 0;
      if (r < k) top[r] = key;
    }
  } else {
#pragma unroll 1
    for (int i = lane; i < L * k; i += kWarp) {
      const int li = i / k;
      const uint64_t key = lists[li * stride + (i - li * k)];
      if (key < T) continue;
      int r = 0;
#pragma unroll 1
      for (int l = 0; l < L; ++l)
#pragma unroll 1
        for (int j = 0; j < k; ++j) r += (lists[l * stride + j] > key) ? 1 : 0;
      if (r < k) top[r] = key;
    }
  }
  __syncwarp();
}

// One warp: the k largest keys of L <= 32 sorted lists (list i at lists +
// i stride, k keys each, descending; keys unique), by a k-way merge: lane i
// holds list i's head; each step takes the largest head (a warp maximum of
// the upper 32 bits, then of the lower ones among those that hold it) into
// top[step], and its lane moves to the next key.  Empty keys (value bits 0)
// sit below every real key, exhausted lists below them.
__device__ __forceinline__ void warp_kway_topk(const uint64_t* lists, int L, int stride, int k, uint64_t* top) {
  const int lane = threadIdx.x & 31;
  int ptr = 0;
  uint64_t head = (lane < L) ? lists[lane * stride] : 0ull;
#pragma unroll 1
  for (int r = 0; r < k; ++r) {
    const uint32_t hi = static_cast<uint32_t>(head >> 32), lo = static_cast<uint32_t>(head);
    const uint32_t mhi = __reduce_max_sync(0xFFFFFFFFu, hi);
    const uint32_t mlo = __reduce_max_sync(0xFFFFFFFFu, hi == mhi ? lo : 0u);
    if (hi == mhi && lo == mlo) {
      top[r] = head;
      ++ptr;
      head = (ptr < k) ? lists[lane * stride + ptr] : 0ull;
    }
  }
  __syncwarp();
}

// Consumer of a sequence whose records fit shared memory (F chunks (k + 2)
// words <= kRecBuf): the records are copied in once every word carries the
// tag (a bounded wait), then one warp per row merges them.  Returns false
// (every thread) if the wait ran out.
__device__ bool consume_smem(const ExpandParams& p, ExpandShared& sh, int b, int base, int64_t nb,
                             const ConsumerPrefetch& pf) {
  constexpr int kPer = (kRecBuf + kNT - 1) / kNT;  // words per thread
  const int tid = threadIdx.x, warp = tid >> 5;
  const int F = p.F;
  const int words = F * p.chunks * (p.k + 2);
  const uint64_t* src = seq_records(p, b);
  const uint32_t tag = static_cast<uint32_t>(p.level) + p.tag_offset;
  ConsumerShared& co = sh.u.co;
  if (tid < F) load_parent(p, pf, b, nb, co);
  uint32_t pending = (1u << kPer) - 1u;  // the thread's words not yet copied
  const uint64_t t0 = tc::globaltimer();
  for (;;) {
    // all loads are in flight before the first is checked
    uint64_t x[kPer];
#pragma unroll
    for (int i = 0; i < kPer; ++i) {
      const int w = tid + i * kNT;
      x[i] = 0ull;
      if (w < words && ((pending >> i) & 1u)) x[i] = ld_relaxed(src + w);
    }
    bool ok = true;
#pragma unroll
    for (int i = 0; i < kPer; ++i) {
      const int w = tid + i * kNT;
      if (w < words && ((pending >> i) & 1u)) {
        if (word_tag(x[i]) == tag) {
          co.rec[w] = x[i];
          pending &= ~(1u << i);
        } else {
          ok = false;
        }
      }
    }
    if (__syncthreads_and(ok)) break;
    if (__syncthreads_or(tc::globaltimer() - t0 > p.wait_limit_ns)) {
      if (tid == 0) flag_error(p.err, LTD_DEVERR_TIMEOUT);
      return false;
    }
    __nanosleep(32);
  }
  // ---- one warp per row: its top k and its log-sum-exp
  const int k = p.k, C = p.chunks, rw = k + 2;
  for (int f = warp; f < F; f += kNW) {
    const uint64_t* row = &co.rec[f * C * rw];
    if (C <= kWarp)
      warp_kway_topk(row, C, rw, k, &co.top[f * k]);
    else
      warp_topk_lists(row, C, rw, k, 0, &co.vals[f * kWarp], co.cand[f], &co.top[f * k]);
    const float lse = row_lse(row, C, rw, k);
    if ((tid & 31) == 0) co.lse[f] = lse;
  }
  __syncthreads();
  // ---- the children, a thread each
  for (int i = tid; i < F * k; i += kNT) {
    const int f = i / k;
    write_child(p, co, nb, base, f, i - f * k, co.top[i]);
  }
  if (tid < F) {
    p.xrow[nb + co.parent[tid]] = static_cast<int32_t>(draft_row(p, tid));
    p.xlse[nb + co.parent[tid]] = co.lse[tid];
  }
  __syncthreads();
  return true;
}

// Large shapes, one warp and one row: waits until items [c0, c0 + n) of the
// row have their records (every word tagged), then merges their key lists
// into `v` (lane i = i-th largest so far) and their (max, sum of exp) into
// (M, S).  Returns false if the wait ran out.
__device__ __forceinline__ bool merge_records(const ExpandParams& p, const uint64_t* row_rec, int c0, int n,
                                           uint64_t& v, float& M, float& S) {
  const int lane = threadIdx.x & 31;
  const int k = p.k, rw = k + 2;
  const uint32_t tag = static_cast<uint32_t>(p.level) + p.tag_offset;
  uint64_t w[kBatch];
  uint64_t s0 = 0ull, s1 = 0ull;
  const uint64_t t0 = tc::globaltimer();
  for (;;) {
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
      w[j] = 0ull;
      if (j < n && lane < k) w[j] = ld_relaxed(row_rec + static_cast<int64_t>(c0 + j) * rw + lane);
    }
    if (lane < n) {
      s0 = ld_relaxed(row_rec + static_cast<int64_t>(c0 + lane) * rw + k);
      s1 = ld_relaxed(row_rec + static_cast<int64_t>(c0 + lane) * rw + k + 1);
    }
    bool ok = true;
#pragma unroll
    for (int j = 0; j < kBatch; ++j)
      if (j < n && lane < k && word_tag(w[j]) != tag) ok = false;
    if (lane < n && (word_tag(s0) != tag || word_tag(s1) != tag)) ok = false;
    if (__all_sync(0xFFFFFFFFu, ok)) break;
    if (tc::globaltimer() - t0 > p.wait_limit_ns) return false;
    __nanosleep(32);
  }
#pragma unroll 1
  for (int j = 0; j < n; ++j) v = (c0 == 0 && j == 0) ? w[0] : warp_merge_desc(v, w[j]);
  float m = lane < n ? stat_float(s0) : -CUDART_INF_F;
  float s = lane < n ? stat_float(s1) : 0.f;
  warp_ms(m, s);
  ms_merge(M, S, m, s);
  return true;
}

// Consumer of a larger sequence: one warp per row merges the row's item
// lists.  Returns false (every thread) if a wait ran out.
__device__ bool consume_warps(const ExpandParams& p, ExpandShared& sh, int b, int base, int64_t nb,
                              const ConsumerPrefetch& pf) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int k = p.k, F = p.F, C = p.chunks;
  ConsumerShared& co = sh.u.co;
  if (tid == 0) sh.h.fail = 0;
  if (tid < F) load_parent(p, pf, b, nb, co);
  __syncthreads();
  for (int f = warp; f < F; f += kNW) {
    const uint64_t* row_rec = seq_records(p, b) + static_cast<int64_t>(f) * C * (k + 2);
    uint64_t v = 0ull;
    float M = -CUDART_INF_F, S = 0.f;
    bool ok = true;
    for (int c0 = 0; c0 < C && ok; c0 += kBatch) ok = merge_records(p, row_rec, c0, min(kBatch, C - c0), v, M, S);
    if (!ok) {
      if (lane == 0) {
        sh.h.fail = 1;
        flag_error(p.err, LTD_DEVERR_TIMEOUT);
      }
      continue;
    }
    // one value for the whole row: tied children get bit-identical cums
    if (lane == 0) co.lse[f] = M + __logf(S);
    __syncwarp();
    if (lane < k) write_child(p, co, nb, base, f, lane, v);
    if (lane == 0) {
      p.xrow[nb + co.parent[f]] = static_cast<int32_t>(draft_row(p, f));
      p.xlse[nb + co.parent[f]] = co.lse[f];
    }
  }
  __syncthreads();
  return sh.h.fail == 0;
}

// Consumer CTA, one sequence: rows merged, children written, the frontier
// chosen.  Every thread of the CTA calls it.
template <bool kLarge>
__device__ void consume_sequence(const ExpandParams& p, ExpandShared& sh, int b, const ConsumerPrefetch& pf) {
  const int tid = threadIdx.x;
  const int k = p.k, F = p.F;
  __syncthreads();  // the producer's last reads of the shared buffers are done
  if (!(pf.b == b ? pf.act != 0 : seq_active(p, b))) return;
  if ((pf.b == b ? pf.lev : __ldcg(&p.n_levels[b])) != p.level - 1) {
    if (tid == 0) flag_error(p.err, LTD_DEVERR_LEVEL);
    return;
  }
  const int64_t nb = static_cast<int64_t>(b) * p.max_nodes;
  const int base = (p.level == 1) ? 1 : 1 + k + (p.level - 2) * k * k;
  bool ok;
  if constexpr (kLarge)
    ok = consume_warps(p, sh, b, base, nb, pf);
  else
    ok = consume_smem(p, sh, b, base, nb, pf);
  TRACE(5);
  if (!ok) return;  // the level stays unbuilt (n_levels unchanged)
  ConsumerShared& co = sh.u.co;
  if (p.level == 1) {
    if (tid < k) p.frontier[b * k + tid] = 1 + tid;
  } else {
    // the k best of the F k children (each row's list is sorted): a k-way
    // merge in warp 0
    if ((tid >> 5) == 0) {
      warp_kway_topk(co.child, F, k, k, co.top);
      if (tid < k) p.frontier[b * k + tid] = static_cast<int32_t>(key_index(co.top[tid]));
    }
  }
  if (tid == 0) {
    p.n_nodes[b] = base + F * k;
    p.n_levels[b] = p.level;
    TRACE(6);
  }
}

// -------------------------------------------------------------------- kernel
template <typename T, bool kLarge>
__global__ void __launch_bounds__(kNT, 2) expand_kernel(const ExpandParams p) {
  extern __shared__ __align__(128) unsigned char expand_smem[];
  ExpandShared& sh = *reinterpret_cast<ExpandShared*>(expand_smem);
  const int tid = threadIdx.x;
  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) tc::mbar_init(tc::smem_u32(&sh.h.bar[s]), 1);
    tc::mbar_init_fence();
    sh.h.n_cand[0] = 0;
    sh.h.n_cand[1] = 0;
    sh.h.load_fail = 0;
  }
  grid_wait();
  trigger_dependents();
  TRACE(0);
  const int i0 = static_cast<int>(blockIdx.x) * p.items_per_cta;
  const int i1 = min(i0 + p.items_per_cta, p.n_items);
  // the sequences whose last item is ours, b_lo..b_hi, are merged after the
  // items; b_lo's flags and frontier are fetched now (loads in volatile asm
  // are issued here, not where first used)
  const int per_seq = p.F * p.chunks;
  const int b_lo = (i0 + per_seq) / per_seq - 1, b_hi = i1 / per_seq - 1;
  ConsumerPrefetch pf{-1, 1, 0, 0, 0.f};
  if (b_lo <= b_hi) {
    pf.b = b_lo;
    pf.act = (p.active == nullptr) ? 1 : ld_cg_early(p.active + b_lo);
    pf.lev = ld_cg_early(&p.n_levels[b_lo]);
    if (p.level > 1 && tid < p.F) pf.parent = ld_cg_early(&p.frontier[b_lo * p.k + tid]);
  }
  // the first items' bytes are requested at once; each later item's when its
  // buffer has been read
  Item qi = item_at(p, i0);  // next to request (thread 0)
  Item qp = qi;              // next to reduce
  if (tid == 0)
    for (int s = 0; s < kStages && i0 + s < i1; ++s) {
      issue_item<T>(p, sh, s, qi);
      advance(p, qi);
    }
  __syncthreads();
  // (records only for sequences at the right level: the consumer flags the
  // rest; each item's level word is read one item ahead)
  int lev = ld_cg_early(&p.n_levels[qp.b]);
  int parity = 0;
  for (int it = i0, n = 0; it < i1; ++it, ++n) {
    const int s = n % kStages;
    Item qn = qp;
    advance(p, qn);
    const int lev_next = (it + 1 < i1) ? ld_cg_early(&p.n_levels[qn.b]) : 0;
    const bool on = sh.h.stage_on[s] != 0;
    // (the parent's cum once its id is in, while the first item loads)
    if (n == 0 && pf.b >= 0 && p.level > 1 && tid < p.F)
      pf.cum = __int_as_float(ld_cg_early(reinterpret_cast<const int32_t*>(
          &p.cum[static_cast<int64_t>(pf.b) * p.max_nodes + pf.parent])));
    if (on) {
      if (!tc::mbar_wait(tc::smem_u32(&sh.h.bar[s]), static_cast<uint32_t>(n / kStages) & 1u)) {
        sh.h.load_fail = 1;
        flag_error(p.err, LTD_DEVERR_TIMEOUT);
      }
      produce_item<T>(p, sh, qp, reinterpret_cast<const T*>(&sh.u.pr.ring[s][0]), lev == p.level - 1, parity);
      parity ^= 1;
      if (n == 0) TRACE(2);
    }
    // every thread has read buffer s (the item's barriers, or this one)
    if (!on) __syncthreads();
    if (tid == 0 && it + kStages < i1) {
      issue_item<T>(p, sh, s, qi);
      advance(p, qi);
    }
    qp = qn;
    lev = lev_next;
  }
  TRACE(3);
  for (int b = b_lo; b <= b_hi; ++b) consume_sequence<kLarge>(p, sh, b, pf);
}

}  // namespace

VocabSplit vocab_split(int64_t rows, int64_t vocab, int64_t target_ctas, int64_t min_elems) {
  rows = rows < 1 ? 1 : rows;
  int64_t chunks = (target_ctas + rows - 1) / rows;
  const int64_t cap = (vocab + min_elems - 1) / min_elems;
  if (chunks > cap) chunks = cap;
  if (chunks < 1) chunks = 1;
  int64_t elems = (vocab + chunks - 1) / chunks;
  elems = (elems + 7) / 8 * 8;
  chunks = (vocab + elems - 1) / elems;
  return VocabSplit{static_cast<int32_t>(chunks), elems};
}

// Items per row the records are sized for (the smaller, fp32, item).
int32_t expand_rec_chunks(int64_t max_vocab) {
  const int64_t v = max_vocab < kExpandMaxVocab ? max_vocab : kExpandMaxVocab;
  const int64_t item = kItemBytes / 4;
  return static_cast<int32_t>((v + item - 1) / item);
}

// Records: batch x k rows x items x (k + 2) words, 256-byte aligned.
size_t expand_scratch_bytes(int32_t batch, int32_t k, int64_t max_vocab) {
  const size_t words = static_cast<size_t>(batch) * k * expand_rec_chunks(max_vocab) * (k + 2);
  return (words * sizeof(uint64_t) + 255) / 256 * 256;
}

cudaError_t launch_tree_reset(const ltd_tree* t, const int32_t* roots, cudaStream_t s) {
  const int threads = 256;
  const int64_t vecs = static_cast<int64_t>(t->scratch_bytes / 16);
  int64_t blocks = (vecs + threads - 1) / threads;
  const int64_t seq_blocks = (t->batch + threads - 1) / threads;
  if (blocks > 2 * static_cast<int64_t>(device_sm_count())) blocks = 2 * static_cast<int64_t>(device_sm_count());
  if (blocks < seq_blocks) blocks = seq_blocks;
  return launch(tree_reset_kernel, dim3(static_cast<unsigned>(blocks)), dim3(threads), 0, s, nullptr, 0,
                *t, roots, static_cast<uint4*>(t->scratch), vecs);
}

// Resident CTAs of one instantiation on this device (the cooperative
// grid's ceiling), computed once.
template <typename T, bool kLarge>
int expand_capacity() {
  static const int cap = [] {
    int per_sm = 0;
    if (cudaFuncSetAttribute(expand_kernel<T, kLarge>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(sizeof(ExpandShared))) != cudaSuccess ||
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, expand_kernel<T, kLarge>, kNT,
                                                      sizeof(ExpandShared)) != cudaSuccess ||
        per_sm < 1)
      per_sm = 1;
    return per_sm * device_sm_count();
  }();
  return cap;
}

template <typename T, bool kLarge>
cudaError_t launch_t(const ExpandParams& params, cudaStream_t s) {
  ExpandParams p = params;
  const int64_t cap = expand_capacity<T, kLarge>();
  int64_t grid = p.n_items < cap ? p.n_items : cap;
  if (grid < 1) grid = 1;
  const int64_t per = (p.n_items + grid - 1) / grid;
  p.items_per_cta = static_cast<int32_t>(per);
  grid = (p.n_items + per - 1) / per;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  return launch(expand_kernel<T, kLarge>, dim3(static_cast<unsigned>(grid)), dim3(kNT), sizeof(ExpandShared),
                s, attr, 1, p);
}

// Leading keys per list for the merge threshold of L sorted k-lists: the
// most that fit a warp (at most k), if L of them reach k; else 0.
int32_t leading_keys(int L, int k) {
  if (L < 1 || L > kWarp) return 0;
  int J = kWarp / L;
  if (J > k) J = k;
  return (J * L >= k) ? J : 0;
}

std::mutex g_expand_hook_mu;
ExpandWaitHook g_expand_hook{};

void set_expand_wait_hook(const ExpandWaitHook& h) {
  std::lock_guard<std::mutex> lock(g_expand_hook_mu);
  g_expand_hook = h;
}

cudaError_t launch_expand(const ExpandParams& params, ltd_dtype dtype, cudaStream_t s) {
  ExpandParams p = params;
  p.item_elems = kItemBytes / (dtype == LTD_BF16 ? 2 : 4);
  p.chunks = static_cast<int32_t>((p.vocab + p.item_elems - 1) / p.item_elems);
  const int64_t n_items = static_cast<int64_t>(p.batch) * p.F * p.chunks;
  if (n_items > 0x7FFFFFFF) return cudaErrorInvalidValue;
  p.n_items = static_cast<int32_t>(n_items);
  ExpandWaitHook h;
  {
    std::lock_guard<std::mutex> lock(g_expand_hook_mu);
    h = g_expand_hook;
  }
  p.wait_limit_ns = h.limit_ns != 0 ? h.limit_ns : tc::kWaitLimitNs;
  p.tag_offset = h.tag_offset;
  p.j_row = leading_keys(p.chunks, p.k);
  const bool large = static_cast<int64_t>(p.F) * p.chunks * (p.k + 2) > kRecBuf;
  if (dtype == LTD_BF16)
    return large ? launch_t<__nv_bfloat16, true>(p, s) : launch_t<__nv_bfloat16, false>(p, s);
  return large ? launch_t<float, true>(p, s) : launch_t<float, false>(p, s);
}

#ifdef LTD_TRACE
extern "C" int ltd_expand_trace_read(unsigned long long* host, int n) {
  return cudaMemcpyFromSymbol(host, g_expand_trace, sizeof(unsigned long long) * n) == cudaSuccess
             ? 0
             : 1;
}
extern "C" int ltd_expand_trace_clear() {
  static unsigned long long zeros[4096 * 8];
  return cudaMemcpyToSymbol(g_expand_trace, zeros, sizeof(zeros)) == cudaSuccess ? 0 : 1;
}
#endif

}  // namespace ltd
