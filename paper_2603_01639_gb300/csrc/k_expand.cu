// Draft tree generation (LTD section 3.2, "Draft Tree Generation").
//
// One launch builds one level for every active sequence.  The grid is
// (chunks, F, batch) with F = 1 at level 1 and F = k afterwards: each CTA
// scans one vocabulary chunk of one frontier row with 16-byte streaming loads,
// computing the chunk's (max, sum exp) and, per thread, its four best
// (logit desc, token asc) keys; bitonic warp networks turn those into the
// chunk's top-k (with an exact rescan in the rare case a thread may hold
// more than four of them).  The last CTA to finish a row (atomic ticket; nothing spins)
// merges the chunk partials in a fixed order into the row's log-sum-exp and
// top-k, appends the k children with cum = cum(parent) + x - lse, and the
// last row of a sequence picks the new frontier: the k best of the k^2 pool
// by (cum desc, node id asc).  Tickets are reset to zero by their last user,
// so the scratch is ready for the next launch.
#include "ltd_common.cuh"
#include "ltd_internal.h"

namespace ltd {

namespace {

constexpr int kNT = 256;

__global__ void tree_reset_kernel(ltd_tree t, const int32_t* __restrict__ roots,
                                  uint32_t* row_ticket, uint32_t* seq_ticket) {
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
  for (int i = 0; i < t.k; ++i) {
    t.frontier[b * t.k + i] = (i == 0) ? 0 : -1;
    row_ticket[b * t.k + i] = 0u;
  }
  seq_ticket[b] = 0u;
}

template <typename T>
__global__ void __launch_bounds__(kNT) expand_kernel(const ExpandParams p) {
  constexpr int NW = kNT / kWarp;
  constexpr int VEC = 16 / sizeof(T);
  constexpr int U = 4;
  __shared__ float red[2 * NW];
  __shared__ uint64_t stage[NW * kWarp];
  __shared__ uint64_t best[kWarp];
  __shared__ int s_last;

  const int ch = blockIdx.x, f = blockIdx.y, b = blockIdx.z, tid = threadIdx.x;
  const int lane = tid & 31, warp = tid >> 5;
  if (p.active != nullptr && p.active[b] == 0) return;
  if (p.n_levels[b] != p.level - 1) {
    if (tid == 0 && ch == 0 && f == 0) flag_error(p.err, LTD_DEVERR_LEVEL);
    return;
  }

  // ---- phase 1: this CTA's chunk of row (b, f)
  const int64_t row = (p.level == 1) ? 0 : 1 + static_cast<int64_t>(p.level - 2) * p.k + f;
  const T* x = reinterpret_cast<const T*>(p.rows) +
               (static_cast<int64_t>(b) * p.rows_per_seq + row) * p.vocab;
  const int64_t lo = static_cast<int64_t>(ch) * p.chunk_elems;
  const int64_t hi = min(lo + p.chunk_elems, p.vocab);

  float m = -CUDART_INF_F, s = 0.f;
  Top4 t4;
  t4.init();
  for (int64_t base = lo + static_cast<int64_t>(tid) * VEC; base < hi;
       base += static_cast<int64_t>(kNT) * VEC * U) {
    float xv[U][VEC];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int64_t i = base + static_cast<int64_t>(u) * kNT * VEC;
      if (i + VEC <= hi) {
        unpack16(ld_stream16(x + i), xv[u], static_cast<const T*>(nullptr));
      } else {
#pragma unroll
        for (int j = 0; j < VEC; ++j) xv[u][j] = (i + j < hi) ? to_f<T>(x[i + j]) : -CUDART_INF_F;
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int64_t i = base + static_cast<int64_t>(u) * kNT * VEC;
      float vm = -CUDART_INF_F;
#pragma unroll
      for (int j = 0; j < VEC; ++j) vm = fmaxf(vm, xv[u][j]);
      if (vm > m) {
        s *= __expf(m - vm);
        m = vm;
      }
#pragma unroll
      for (int j = 0; j < VEC; ++j) {
        if (i + j < hi) {
          const float xj = xv[u][j];
          s += (xj == -CUDART_INF_F) ? 0.f : __expf(xj - m);
          t4.insert(make_key(xj, static_cast<uint32_t>(i + j)));
        }
      }
    }
  }
  block_ms<kNT>(m, s, red);
  // warp lists from the per-thread top-4s, then the block list
  WarpTopK wt;
  wt.init();
  wt.offer(t4.t0, p.k);
  wt.offer(t4.t1, p.k);
  wt.offer(t4.t2, p.k);
  wt.offer(t4.t3, p.k);
  block_topk<kNT>(wt, stage, best);
  // exactness: a thread whose 4th key made the top-k may hold more of it;
  // then every thread offers its whole chunk again (rare: needs 4 of the
  // chunk's top-k in one thread's 1/256 of the chunk)
  if (__syncthreads_or(t4.t3 != 0ull && t4.t3 >= best[p.k - 1])) {
    wt.init();
    for (int64_t wbase = lo + static_cast<int64_t>(warp) * kWarp; wbase < hi;
         wbase += static_cast<int64_t>(kNT)) {
      const int64_t i = wbase + lane;
      wt.offer(i < hi ? make_key(to_f<T>(x[i]), static_cast<uint32_t>(i)) : 0ull, p.k);
    }
    block_topk<kNT>(wt, stage, best);
  }

  const int64_t rec_row = (static_cast<int64_t>(b) * p.F + f) * p.chunks;
  if (tid == 0) p.part_ms[rec_row + ch] = make_float2(m, s);
  if (tid < p.k) p.part_keys[(rec_row + ch) * p.k + tid] = best[tid];
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    const uint32_t prev = atomicAdd(&p.row_ticket[b * p.k + f], 1u);
    s_last = (prev == static_cast<uint32_t>(p.chunks - 1));
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();

  // ---- phase 2: last CTA of the row merges its chunks (fixed order)
  float M = -CUDART_INF_F, S = 0.f;
  for (int c = tid; c < p.chunks; c += kNT) {
    const float2 ms = __ldcg(&p.part_ms[rec_row + c]);
    ms_merge(M, S, ms.x, ms.y);
  }
  block_ms<kNT>(M, S, red);
  WarpTopK t2;
  t2.init();
  for (int c = warp; c < p.chunks; c += NW)
    t2.merge_sorted(lane < p.k ? __ldcg(&p.part_keys[(rec_row + c) * p.k + lane]) : 0ull);
  block_topk<kNT>(t2, stage, best);
  const float lse = M + logf(S);

  const int64_t nb = static_cast<int64_t>(b) * p.max_nodes;
  const int parent = (p.level == 1) ? 0 : __ldcg(&p.frontier[b * p.k + f]);
  const float cum_p = (p.level == 1) ? 0.f : __ldcg(&p.cum[nb + parent]);
  const int base = (p.level == 1) ? 1 : 1 + p.k + (p.level - 2) * p.k * p.k;
  if (tid < p.k) {
    const uint64_t key = best[tid];
    const int64_t id = nb + base + f * p.k + tid;
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
    p.row_ticket[b * p.k + f] = 0u;
  }
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    const uint32_t prev = atomicAdd(&p.seq_ticket[b], 1u);
    s_last = (prev == static_cast<uint32_t>(p.F - 1));
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();

  // ---- phase 3: last row of the sequence picks the frontier
  if (p.level == 1) {
    if (tid < p.k) p.frontier[b * p.k + tid] = 1 + tid;
  } else {
    WarpTopK t3;
    t3.init();
    const int pool = p.k * p.k;
    for (int j0 = warp * kWarp; j0 < pool; j0 += kNT) {
      const int j = j0 + lane;
      const int id = base + j;
      t3.offer(j < pool ? make_key(__ldcg(&p.cum[nb + id]), static_cast<uint32_t>(id)) : 0ull, p.k);
    }
    block_topk<kNT>(t3, stage, best);
    if (tid < p.k) p.frontier[b * p.k + tid] = static_cast<int32_t>(key_index(best[tid]));
  }
  if (tid == 0) {
    p.n_nodes[b] = base + p.F * p.k;
    p.n_levels[b] = p.level;
    p.seq_ticket[b] = 0u;
  }
}

template <typename T>
cudaError_t launch_expand_t(const ExpandParams& p, int32_t batch, cudaStream_t s) {
  const dim3 grid(p.chunks, p.F, batch);
  expand_kernel<T><<<grid, kNT, 0, s>>>(p);
  return cudaGetLastError();
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

ExpandRecordLayout expand_layout(int32_t batch, int32_t k, int64_t max_vocab) {
  ExpandRecordLayout l{};
  const int64_t r1 = static_cast<int64_t>(batch) *
                     vocab_split(batch, max_vocab, kExpandTargetCtas, kExpandMinElems).chunks;
  const int64_t rk = static_cast<int64_t>(batch) * k *
                     vocab_split(static_cast<int64_t>(batch) * k, max_vocab, kExpandTargetCtas,
                                 kExpandMinElems).chunks;
  l.records = r1 > rk ? r1 : rk;
  auto up = [](size_t x) { return (x + 255) / 256 * 256; };
  l.ms_bytes = up(l.records * sizeof(float2));
  l.keys_bytes = up(l.records * k * sizeof(uint64_t));
  l.row_ticket_bytes = up(static_cast<size_t>(batch) * k * sizeof(uint32_t));
  l.seq_ticket_bytes = up(static_cast<size_t>(batch) * sizeof(uint32_t));
  l.total = l.ms_bytes + l.keys_bytes + l.row_ticket_bytes + l.seq_ticket_bytes;
  return l;
}

cudaError_t launch_tree_reset(const ltd_tree* t, const int32_t* roots, cudaStream_t s) {
  const ExpandRecordLayout l = expand_layout(t->batch, t->k, t->max_vocab);
  char* base = static_cast<char*>(t->scratch);
  uint32_t* row_ticket = reinterpret_cast<uint32_t*>(base + l.ms_bytes + l.keys_bytes);
  uint32_t* seq_ticket = reinterpret_cast<uint32_t*>(base + l.ms_bytes + l.keys_bytes +
                                                     l.row_ticket_bytes);
  const int threads = 128;
  tree_reset_kernel<<<(t->batch + threads - 1) / threads, threads, 0, s>>>(*t, roots, row_ticket,
                                                                            seq_ticket);
  return cudaGetLastError();
}

cudaError_t launch_expand(const ExpandParams& p, int32_t batch, ltd_dtype dtype, cudaStream_t s) {
  return dtype == LTD_BF16 ? launch_expand_t<__nv_bfloat16>(p, batch, s)
                           : launch_expand_t<float>(p, batch, s);
}

}  // namespace ltd
