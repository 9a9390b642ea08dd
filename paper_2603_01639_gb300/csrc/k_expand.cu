// Draft tree generation (LTD section 3.2, "Draft Tree Generation").
//
// One launch builds one level for every active sequence.  The grid is
// (C, F, batch): F = 1 row at level 1, F = k rows (one per frontier node)
// afterwards, and each row is split into C <= 8 vocabulary chunks whose CTAs
// form one thread-block cluster.
//
// Per CTA (chunk): every thread loads its elements into registers with
// 16-byte streaming loads and computes its own max and sum of exp -- no
// per-element branches.  The k-th largest of the per-thread maxima, T, is a
// lower bound of the chunk's k-th largest logit (at least k threads hold an
// element >= T), so only elements >= T can be in the chunk's top-k: they
// (typically about k of them) are appended to a shared list and ranked
// exactly by (logit desc, token asc) with bitonic warp networks.  Inputs
// that make that list overflow (huge tie sets) fall back to an exact
// re-offer of the whole chunk.
// Per row: rank 0 of the cluster gathers its peers' chunk lists and
// (max, sum exp) through distributed shared memory, merges them, and
// appends the k children with cum = cum(parent) + x - logsumexp(row) (fp32).
// Per sequence: the last row to finish (one atomic ticket, nothing spins)
// selects the new frontier: the k best of the k^2 children by (cum desc,
// node id asc).  The ticket is reset by its last user.
#include "ltd_common.cuh"
#include "ltd_internal.h"
#include "tc_util.cuh"

namespace ltd {

namespace {

constexpr int kNT = 512;
constexpr int kNW = kNT / kWarp;
constexpr int kCand = 512;   // candidate list capacity per chunk
constexpr int kMaxChunks = 8;
constexpr int kMaxVec = 8;   // 16-byte vectors per thread

// Optional phase timestamps for performance work (off in normal builds).
#ifdef LTD_TRACE
__device__ unsigned long long g_expand_trace[4096][16];
#define TRACE(slot)                                                                  \
  do {                                                                               \
    const int cta_ = blockIdx.x + gridDim.x * (blockIdx.y + gridDim.y * blockIdx.z); \
    unsigned long long t_;                                                           \
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t_));                          \
    if (cta_ < 4096) g_expand_trace[cta_][slot] = t_;                                \
  } while (0)
#else
#define TRACE(slot) \
  do {              \
  } while (0)
#endif

__global__ void tree_reset_kernel(ltd_tree t, const int32_t* __restrict__ roots,
                                  uint32_t* seq_ticket) {
  grid_wait();
  trigger_dependents();
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= t.batch) return;
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
  seq_ticket[b] = 0u;
}

// Warp bitonic sort of one float per lane, descending (lane 0 = largest).
__device__ __forceinline__ float warp_sort_desc_f(float v) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int size = 2; size <= 32; size <<= 1) {
#pragma unroll
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      const float o = __shfl_xor_sync(0xFFFFFFFFu, v, stride);
      const bool keep_max = ((lane & stride) == 0) == ((lane & size) == 0);
      v = keep_max ? fmaxf(v, o) : fminf(v, o);
    }
  }
  return v;
}
// Tree merge of one descending 32-entry list per warp (stage[w][lane]) into
// stage[0][0..32).  All threads call; returns after a barrier.
template <typename V, V (*Merge)(V, V)>
__device__ __forceinline__ void tree_merge(V* stage) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll 1
  for (int step = 1; step < kNW; step <<= 1) {
    __syncthreads();
    if ((warp % (2 * step)) == 0 && warp + step < kNW) {
      const V m = Merge(stage[warp * kWarp + lane], stage[(warp + step) * kWarp + lane]);
      __syncwarp();
      stage[warp * kWarp + lane] = m;
    }
  }
  __syncthreads();
}

// Raw bits of element i of x, or of -inf past the end.
__device__ __forceinline__ uint32_t raw_or_ninf(const float* x, int64_t i, int64_t hi) {
  return i < hi ? __float_as_uint(x[i]) : 0xFF800000u;
}
__device__ __forceinline__ uint32_t raw_or_ninf(const __nv_bfloat16* x, int64_t i, int64_t hi) {
  return i < hi ? static_cast<uint32_t>(__bfloat16_as_ushort(x[i])) : 0xFF80u;
}
template <typename T>
__device__ __forceinline__ uint4 load_tail(const T* x, int64_t i, int64_t hi) {
  uint32_t w[4];
  if constexpr (sizeof(T) == 4) {
#pragma unroll
    for (int q = 0; q < 4; ++q) w[q] = raw_or_ninf(x, i + q, hi);
  } else {
#pragma unroll
    for (int q = 0; q < 4; ++q)
      w[q] = raw_or_ninf(x, i + 2 * q, hi) | (raw_or_ninf(x, i + 2 * q + 1, hi) << 16);
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}
struct ExpandShared {
  uint64_t stage[kNW * kWarp];
  float fstage[kNW * kWarp];
  uint64_t cand[kCand];
  float red[2 * kNW + 1];
  // published to the cluster: the chunk's sorted top list and (max, sum exp)
  uint64_t top[kWarp];
  float2 ms;
  // gathered by rank 0
  uint64_t peer_top[kMaxChunks][kWarp];
  float2 peer_ms[kMaxChunks];
  float thr;
  int n_cand;
  int wcnt[kNW];
  int last;
};

template <typename T, int U>
__global__ void __launch_bounds__(kNT) expand_kernel(const ExpandParams p) {
  constexpr int VEC = 16 / sizeof(T);
  __shared__ ExpandShared sh;
  grid_wait();
  trigger_dependents();
  const int ch = blockIdx.x, f = blockIdx.y, b = blockIdx.z, tid = threadIdx.x;
  const int lane = tid & 31, warp = tid >> 5;
  if (tid == 0) TRACE(0);
  // early exits are shared by the whole cluster (same row)
  if (p.active != nullptr && p.active[b] == 0) return;
  if (p.n_levels[b] != p.level - 1) {
    if (tid == 0 && ch == 0 && f == 0) flag_error(p.err, LTD_DEVERR_LEVEL);
    return;
  }
  const int k = p.k;

  // ---- stage 1: chunk elements into registers; per-thread max and sum exp
  const int64_t row = (p.level == 1) ? 0 : 1 + static_cast<int64_t>(p.level - 2) * k + f;
  const T* x = reinterpret_cast<const T*>(p.rows) +
               (static_cast<int64_t>(b) * p.rows_per_seq + row) * p.vocab;
  const int64_t lo = static_cast<int64_t>(ch) * p.chunk_elems;
  const int64_t hi = min(lo + p.chunk_elems, p.vocab);
  // the chunk stays in registers as loaded (16 bytes per vector) and is
  // unpacked where it is used
  uint4 raw[U];
#pragma unroll
  for (int u = 0; u < U; ++u) {
    const int64_t i = lo + (static_cast<int64_t>(u) * kNT + tid) * VEC;
    raw[u] = (i + VEC <= hi) ? ld_stream16_once(x + i) : load_tail(x, i, hi);
  }
  float tmax = -CUDART_INF_F;
#pragma unroll
  for (int u = 0; u < U; ++u)
#pragma unroll
    for (int j = 0; j < VEC; ++j) tmax = fmaxf(tmax, elem<T>(raw[u], j));
  float tsum = 0.f;
  if (tmax > -CUDART_INF_F) {
#pragma unroll
    for (int u = 0; u < U; ++u)
#pragma unroll
      for (int j = 0; j < VEC; ++j) tsum += __expf(elem<T>(raw[u], j) - tmax);
  }
  if (tid == 0) TRACE(1);
  // ---- stage 2: T = k-th largest of the 32 half-warp maxima, a lower bound
  // of the chunk's k-th largest logit (k half-warps hold an element >= T);
  // the largest of them is the chunk's max M
  float hm = tmax;
#pragma unroll
  for (int o = 8; o > 0; o >>= 1) hm = fmaxf(hm, __shfl_xor_sync(0xFFFFFFFFu, hm, o));
  if ((lane & 15) == 0) sh.fstage[warp * 2 + (lane >> 4)] = hm;
  __syncthreads();
  if (warp == 0) {
    const float v = warp_sort_desc_f(sh.fstage[lane]);  // 2 * kNW = 32 half-warps
    if (lane == k - 1) sh.thr = v;
    if (lane == 0) sh.red[2 * kNW] = v;  // the chunk max
  }
  if (tid == 0) TRACE(10);
  __syncthreads();
  if (tid == 0) TRACE(11);
  const float thr = sh.thr;
  const float cmax = sh.red[2 * kNW];
  // the chunk's sum of exp(x - cmax): one rescale per thread, then a warp sum
  {
    float e = (tmax > -CUDART_INF_F) ? tsum * __expf(tmax - cmax) : 0.f;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) e += __shfl_xor_sync(0xFFFFFFFFu, e, o);
    if (lane == 0) sh.red[warp] = e;
  }

  // ---- stage 3: the candidates >= T, ranked exactly by (logit desc, token asc);
  // each thread marks its elements >= T, the warps' counts give every
  // thread its slots (no atomics)
  uint64_t cmask = 0ull;
  if (tmax >= thr) {
#pragma unroll
    for (int u = 0; u < U; ++u)
#pragma unroll
      for (int j = 0; j < VEC; ++j) {
        const int64_t i = lo + (static_cast<int64_t>(u) * kNT + tid) * VEC + j;
        if (elem<T>(raw[u], j) >= thr && i < hi) cmask |= 1ull << (u * VEC + j);
      }
  }
  const int cnt = __popcll(cmask);
  int incl = cnt;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
    if (lane >= o) incl += y;
  }
  if (lane == 31) sh.wcnt[warp] = incl;
  __syncthreads();
  {
    int below = (lane < warp) ? sh.wcnt[lane] : 0;  // kNW <= 32 warps
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) below += __shfl_xor_sync(0xFFFFFFFFu, below, o);
    int slot = below + incl - cnt;
    if (cmask != 0ull) {
#pragma unroll
      for (int u = 0; u < U; ++u)
#pragma unroll
        for (int j = 0; j < VEC; ++j)
          if ((cmask >> (u * VEC + j)) & 1ull) {
            const int64_t i = lo + (static_cast<int64_t>(u) * kNT + tid) * VEC + j;
            if (slot < kCand) sh.cand[slot] = make_key(elem<T>(raw[u], j), static_cast<uint32_t>(i));
            ++slot;
          }
    }
  }
  if (tid < kWarp) {
    int t = tid < kNW ? sh.wcnt[tid] : 0;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xFFFFFFFFu, t, o);
    if (tid == 0) sh.n_cand = t;
  }
  __syncthreads();
  if (tid == 0) TRACE(12);
  const int nc = sh.n_cand;
  if (nc <= kCand) {
    // typically a few dozen: one warp ranks them
    if (warp == 0) {
      WarpTopK wt;
      wt.init();
      for (int c0 = 0; c0 < nc; c0 += kWarp) {
        const int c = c0 + lane;
        wt.offer(c < nc ? sh.cand[c] : 0ull, k);
      }
      sh.top[lane] = wt.v;
    }
  } else {
    // exact fallback (huge tie sets): every element of the chunk is offered
    WarpTopK wt;
    wt.init();
#pragma unroll
    for (int u = 0; u < U; ++u)
#pragma unroll
      for (int j = 0; j < VEC; ++j) {
        const int64_t i = lo + (static_cast<int64_t>(u) * kNT + tid) * VEC + j;
        wt.offer(i < hi ? make_key(elem<T>(raw[u], j), static_cast<uint32_t>(i)) : 0ull, k);
      }
    sh.stage[warp * kWarp + lane] = wt.v;
    tree_merge<uint64_t, warp_merge_desc>(sh.stage);
    if (tid < kWarp) sh.top[tid] = sh.stage[tid];
  }
  if (warp == 1) {
    // (max, sum exp) of the chunk from the warps' sums
    float csum = lane < kNW ? sh.red[lane] : 0.f;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) csum += __shfl_xor_sync(0xFFFFFFFFu, csum, o);
    if (lane == 0) sh.ms = make_float2(cmax, csum);
  }
  if (tid == 0) TRACE(2);

  // ---- row: rank 0 gathers the chunk results of its cluster (warp 0 reads
  // every peer's list and merges them) before the barrier that lets the
  // peers leave
  const int C = p.chunks;
  tc::cluster_sync();
  if (ch == 0 && warp == 0) {
    uint64_t lists[kMaxChunks];
#pragma unroll
    for (int c = 0; c < kMaxChunks; ++c)
      lists[c] = c < C ? tc::ld_cluster_u64(tc::mapa(tc::smem_u32(&sh.top[lane]), c)) : 0ull;
    const float2 pm = lane < C ? tc::ld_cluster_f2(tc::mapa(tc::smem_u32(&sh.ms), lane))
                               : make_float2(-CUDART_INF_F, 0.f);
    uint64_t v = lists[0];
#pragma unroll
    for (int c = 1; c < kMaxChunks; ++c)
      if (c < C) v = warp_merge_desc(v, lists[c]);
    sh.stage[lane] = v;
    // (max, sum exp) of the row from the lanes' chunk pairs
    float M = pm.x, S = pm.y;
#pragma unroll
    for (int o = 1; o < kMaxChunks; o <<= 1) {
      const float M2 = __shfl_xor_sync(0xFFFFFFFFu, M, o), S2 = __shfl_xor_sync(0xFFFFFFFFu, S, o);
      ms_merge(M, S, M2, S2);
    }
    if (lane == 0) sh.red[0] = M + logf(S);
  }
  // no CTA leaves while rank 0 may still read its shared memory; the
  // barrier also publishes warp 0's results to the rest of rank 0
  tc::cluster_sync();
  if (ch != 0) return;
  if (tid == 0) TRACE(3);
  if (tid == 0) TRACE(7);
  const float lse = sh.red[0];

  const int64_t nb = static_cast<int64_t>(b) * p.max_nodes;
  const int parent = (p.level == 1) ? 0 : __ldcg(&p.frontier[b * k + f]);
  if (tid == 0) TRACE(8);
  const float cum_p = (p.level == 1) ? 0.f : __ldcg(&p.cum[nb + parent]);
  if (tid == 0) TRACE(9);
  const int base = (p.level == 1) ? 1 : 1 + k + (p.level - 2) * k * k;
  if (tid < k) {
    const uint64_t key = sh.stage[tid];
    const int64_t id = nb + base + f * k + tid;
    p.token[id] = static_cast<int32_t>(key_index(key));
    p.parent[id] = parent;
    p.depth[id] = p.level;
    p.cum[id] = cum_p + (key_value(key) - lse);
    p.xrow[id] = -1;
    p.xlse[id] = 0.f;
  }
  if (tid == 0) {
    p.xrow[nb + parent] = static_cast<int32_t>(row);
    p.xlse[nb + parent] = lse;
    TRACE(4);
  }

  // ---- sequence: the frontier (level 1: all children; later: by the last row)
  if (p.level == 1) {
    if (tid < k) p.frontier[b * k + tid] = 1 + tid;
    if (tid == 0) {
      p.n_nodes[b] = 1 + k;
      p.n_levels[b] = 1;
    }
    return;
  }
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    const uint32_t prev = atomicAdd(&p.seq_ticket[b], 1u);
    sh.last = (prev == static_cast<uint32_t>(p.F - 1));
  }
  __syncthreads();
  if (!sh.last) return;
  __threadfence();
  if (tid == 0) TRACE(5);
  const int pool = k * k;
  if (pool <= 4 * kWarp) {
    // a small pool: one warp, no block barriers
    if (warp == 0) {
      // all of the pool's loads go out before the first is needed
      uint64_t keys[4];
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        const int j = r * kWarp + lane;
        keys[r] = j < pool ? make_key(__ldcg(&p.cum[nb + base + j]), static_cast<uint32_t>(base + j)) : 0ull;
      }
      WarpTopK pt;
      pt.init();
#pragma unroll
      for (int r = 0; r < 4; ++r)
        if (r * kWarp < pool) pt.offer(keys[r], k);
      if (lane < k) p.frontier[b * k + lane] = static_cast<int32_t>(key_index(pt.v));
    }
  } else {
    WarpTopK pt;
    pt.init();
    for (int j0 = warp * kWarp; j0 < pool; j0 += kNT) {
      const int j = j0 + lane;
      const int id = base + j;
      pt.offer(j < pool ? make_key(__ldcg(&p.cum[nb + id]), static_cast<uint32_t>(id)) : 0ull, k);
    }
    sh.stage[warp * kWarp + lane] = pt.v;
    tree_merge<uint64_t, warp_merge_desc>(sh.stage);
    if (tid < k) p.frontier[b * k + tid] = static_cast<int32_t>(key_index(sh.stage[tid]));
  }
  if (tid == 0) {
    p.n_nodes[b] = base + p.F * k;
    p.n_levels[b] = p.level;
    p.seq_ticket[b] = 0u;
    TRACE(6);
  }
}

template <typename T, int U>
cudaError_t launch_u(const ExpandParams& p, int32_t batch, cudaStream_t s) {
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = p.chunks;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  return launch(expand_kernel<T, U>, dim3(p.chunks, p.F, batch), dim3(kNT), 0, s, attr, 1, p);
}

template <typename T>
cudaError_t launch_t(const ExpandParams& p, int32_t batch, cudaStream_t s) {
  constexpr int VEC = 16 / sizeof(T);
  const int64_t vecs = (p.chunk_elems + static_cast<int64_t>(kNT) * VEC - 1) /
                       (static_cast<int64_t>(kNT) * VEC);
  if (vecs <= 1) return launch_u<T, 1>(p, batch, s);
  if (vecs <= 2) return launch_u<T, 2>(p, batch, s);
  if (vecs <= 4) return launch_u<T, 4>(p, batch, s);
  if (vecs <= kMaxVec) return launch_u<T, kMaxVec>(p, batch, s);
  return cudaErrorInvalidValue;
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

int64_t expand_max_vocab(int elem_bytes) {
  return static_cast<int64_t>(kMaxChunks) * kNT * kMaxVec * (16 / elem_bytes);
}

// At most 8 chunks (one cluster) per row of at most 512 threads x 8 vectors.
VocabSplit expand_split(int64_t rows, int64_t vocab, int elem_bytes) {
  const int64_t max_chunk = static_cast<int64_t>(kNT) * kMaxVec * (16 / elem_bytes);
  VocabSplit v = vocab_split(rows, vocab, kExpandTargetCtas, kExpandMinElems);
  if (v.chunks > kMaxChunks || v.chunk_elems > max_chunk) {
    int64_t chunks = (vocab + max_chunk - 1) / max_chunk;
    if (chunks < v.chunks) chunks = v.chunks;
    if (chunks > kMaxChunks) chunks = kMaxChunks;
    int64_t elems = (vocab + chunks - 1) / chunks;
    elems = (elems + 7) / 8 * 8;
    v.chunks = static_cast<int32_t>((vocab + elems - 1) / elems);
    v.chunk_elems = elems;
  }
  return v;
}

ExpandRecordLayout expand_layout(int32_t batch, int32_t k, int64_t max_vocab) {
  (void)k;
  (void)max_vocab;
  ExpandRecordLayout l{};
  l.seq_ticket_bytes = (static_cast<size_t>(batch) * sizeof(uint32_t) + 255) / 256 * 256;
  l.total = l.seq_ticket_bytes;
  return l;
}

cudaError_t launch_tree_reset(const ltd_tree* t, const int32_t* roots, cudaStream_t s) {
  uint32_t* seq_ticket = static_cast<uint32_t*>(t->scratch);
  const int threads = 128;
  return launch(tree_reset_kernel, dim3((t->batch + threads - 1) / threads), dim3(threads), 0, s,
                nullptr, 0, *t, roots, seq_ticket);
}

cudaError_t launch_expand(const ExpandParams& p, int32_t batch, ltd_dtype dtype, cudaStream_t s) {
  return dtype == LTD_BF16 ? launch_t<__nv_bfloat16>(p, batch, s) : launch_t<float>(p, batch, s);
}

#ifdef LTD_TRACE
extern "C" int ltd_expand_trace_read(unsigned long long* host, int n) {
  return cudaMemcpyFromSymbol(host, g_expand_trace, sizeof(unsigned long long) * n) == cudaSuccess
             ? 0
             : 1;
}
extern "C" int ltd_expand_trace_clear() {
  static unsigned long long zeros[4096 * 16];
  return cudaMemcpyToSymbol(g_expand_trace, zeros, sizeof(zeros)) == cudaSuccess ? 0 : 1;
}
#endif

}  // namespace ltd
