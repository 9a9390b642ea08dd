// Acceptance and KV compaction (LTD section 3.2, "Draft Tree Verification").
//
// accept_rows_kernel: grid (chunks, n_max, batch).  Each CTA scans one chunk
// of one verified slot's target row and records (max, sum exp, argmax key)
// in the workspace.
// accept_walk_kernel: one thread-block cluster of C CTAs per sequence.
//  - greedy: rank 0 merges the argmax records (ties to the lower token id),
//    marks every slot whose token is its parent's argmax, and follows those
//    marks from slot 0; the argmax at the end is the bonus token;
//  - stochastic (T = 1): SpecInfer-style multi-candidate speculative
//    sampling.  Each CTA holds one vocabulary slice of p (target) and q
//    (draft) in shared memory.  Child i of the current slot is accepted if
//    r_i q(x_i) < p(x_i) -- every CTA evaluates that test identically --
//    else p <- max(p - q, 0) / Z, with Z summed over the cluster through
//    distributed shared memory (partials added in rank order, so every CTA
//    holds the same Z).  With no child accepted the bonus is a Gumbel-max
//    draw from p, reduced over the cluster the same way.
// kv_compact_kernel: grid (KV heads, layers x {K, V}, batch); each CTA stages
// the accepted rows in shared memory, then writes them to ctx+t, so a row
// that is both a source and a destination is read before it is overwritten.
#include "ltd_common.cuh"
#include "ltd_internal.h"
#include "tc_util.cuh"

namespace ltd {

namespace {

constexpr int kNT = 512;
constexpr int kNW = kNT / kWarp;
constexpr int64_t kSliceMax = 16384;  // vocabulary elements per walk CTA
constexpr int kMaxWalkCluster = static_cast<int>(kAcceptMaxVocab / kSliceMax);

template <typename T>
__global__ void __launch_bounds__(kNT) accept_rows_kernel(const AcceptParams p) {
  constexpr int VEC = 16 / sizeof(T);
  constexpr int U = 2;
  __shared__ float red[2 * kNW];
  __shared__ uint64_t redk[kNW];
  grid_wait();
  trigger_dependents();

  const int ch = blockIdx.x, i = blockIdx.y, b = blockIdx.z, tid = threadIdx.x;
  const int N = p.n_verify[b];
  if (N < 1 || N > p.n_max || i >= N) return;

  const T* row = reinterpret_cast<const T*>(p.target) +
                 (static_cast<int64_t>(b) * p.n_max + i) * p.vocab;
  const int64_t lo = static_cast<int64_t>(ch) * p.chunk_elems;
  const int64_t hi = min(lo + p.chunk_elems, p.vocab);
  float m = -CUDART_INF_F, s = 0.f;
  uint64_t best = 0ull;
  for (int64_t base = lo + static_cast<int64_t>(tid) * VEC; base < hi;
       base += static_cast<int64_t>(kNT) * VEC * U) {
    float xv[U][VEC];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int64_t idx = base + static_cast<int64_t>(u) * kNT * VEC;
      if (idx + VEC <= hi) {
        unpack16(ld_stream16(row + idx), xv[u], static_cast<const T*>(nullptr));
      } else {
#pragma unroll
        for (int j = 0; j < VEC; ++j)
          xv[u][j] = (idx + j < hi) ? to_f<T>(row[idx + j]) : -CUDART_INF_F;
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int64_t idx = base + static_cast<int64_t>(u) * kNT * VEC;
      float vm = -CUDART_INF_F;
      int jm = 0;
#pragma unroll
      for (int j = 0; j < VEC; ++j)
        if (xv[u][j] > vm) {
          vm = xv[u][j];
          jm = j;
        }
      if (vm > m) {
        s *= __expf(m - vm);
        m = vm;
      }
      float add = 0.f;
#pragma unroll
      for (int j = 0; j < VEC; ++j) add += (xv[u][j] == -CUDART_INF_F) ? 0.f : __expf(xv[u][j] - m);
      s += add;
      if (idx < hi) {
        const uint64_t key = make_key(vm, static_cast<uint32_t>(idx + jm));
        best = key > best ? key : best;
      }
    }
  }
  block_ms<kNT>(m, s, red);
  best = block_max_u64<kNT>(best, redk);
  if (tid == 0) {
    AcceptRecord* r = p.rec + (static_cast<int64_t>(b) * p.n_max + i) * p.chunks + ch;
    r->m = m;
    r->s = s;
    r->key = best;
  }
}

struct WalkShared {
  int32_t node[LTD_MAX_N];
  int32_t tok[LTD_MAX_N];
  int32_t pslot[LTD_MAX_N];
  int32_t am[LTD_MAX_N];
  int32_t next[LTD_MAX_N];
  int32_t kids[LTD_MAX_N];
  float Z[LTD_MAX_N];
  int32_t path[LTD_MAX_DEPTH + 1];
  float red[2 * kNW];
  uint64_t redk[kNW];
  float cell_z[2];          // cluster exchange cells, double-buffered by round
  uint64_t cell_key[2];
  float2 cell_ms;
  int n_kids;
};

// Sum of every cluster CTA's `v` (rank order, so all CTAs get the same bits).
__device__ __forceinline__ float cluster_sum(float v, float* cells, int& round, int C) {
  const int c = round & 1;
  if (threadIdx.x == 0) cells[c] = v;
  tc::cluster_sync();
  float t = 0.f;
  for (int r = 0; r < C; ++r) t += tc::ld_cluster_f1(tc::mapa(tc::smem_u32(&cells[c]), r));
  ++round;
  return t;
}
__device__ __forceinline__ uint64_t cluster_max_u64(uint64_t v, uint64_t* cells, int& round,
                                                    int C) {
  const int c = round & 1;
  if (threadIdx.x == 0) cells[c] = v;
  tc::cluster_sync();
  uint64_t t = 0ull;
  for (int r = 0; r < C; ++r) {
    const uint64_t x = tc::ld_cluster_u64(tc::mapa(tc::smem_u32(&cells[c]), r));
    t = x > t ? x : t;
  }
  ++round;
  return t;
}

template <typename T>
__global__ void __launch_bounds__(kNT) accept_walk_kernel(const AcceptParams p, int C,
                                                          int64_t slice) {
  extern __shared__ float dyn[];
  __shared__ WalkShared sh;
  grid_wait();
  trigger_dependents();
  float* ps = dyn;
  float* qs = dyn + slice;
  const int rank = blockIdx.x, b = blockIdx.y, tid = threadIdx.x;
  const int N = p.n_verify[b];
  const int mode = p.mode[b];
  int32_t* path_out = p.path + static_cast<int64_t>(b) * (p.max_depth + 1);
  // everything below is uniform over the cluster (one sequence)
  if (N < 1 || N > p.n_max || (mode != LTD_GREEDY && mode != LTD_STOCHASTIC)) {
    if (rank == 0 && tid == 0) {
      flag_error(p.err, (N < 1 || N > p.n_max) ? LTD_DEVERR_NVERIFY : LTD_DEVERR_MODE);
      for (int t = 0; t <= p.max_depth; ++t) path_out[t] = -1;
      p.accept_len[b] = -1;
      p.bonus[b] = -1;
      p.new_ctx[b] = p.ctx[b];
    }
    return;
  }
  if (mode == LTD_GREEDY && rank != 0) return;

  const int64_t nb = static_cast<int64_t>(b) * p.max_nodes;
  const int64_t V = p.vocab;
  for (int j = tid; j < N; j += kNT) {
    const int nid = p.node_ids[static_cast<int64_t>(b) * p.n_max + j];
    sh.node[j] = nid;
    sh.tok[j] = p.token[nb + nid];
    sh.next[j] = -1;
  }
  __syncthreads();
  for (int j = tid; j < N; j += kNT) {
    const int par = p.parent[nb + sh.node[j]];
    int lo = 0, hi = j - 1, found = -1;  // slots hold ascending node ids
    while (lo <= hi) {
      const int mid = (lo + hi) >> 1;
      const int v = sh.node[mid];
      if (v == par) {
        found = mid;
        break;
      }
      if (v < par) lo = mid + 1;
      else hi = mid - 1;
    }
    sh.pslot[j] = found;
  }
  __syncthreads();
  auto row_lse = [&](int slot) {
    const AcceptRecord* r = p.rec + (static_cast<int64_t>(b) * p.n_max + slot) * p.chunks;
    float M = -CUDART_INF_F, S = 0.f;
    for (int c = 0; c < p.chunks; ++c) ms_merge(M, S, r[c].m, r[c].s);
    return M + logf(S);
  };

  if (mode == LTD_GREEDY) {
    for (int j = tid; j < N; j += kNT) {
      const AcceptRecord* r = p.rec + (static_cast<int64_t>(b) * p.n_max + j) * p.chunks;
      unsigned long long best = 0ull;
      for (int c = 0; c < p.chunks; ++c) best = r[c].key > best ? r[c].key : best;
      sh.am[j] = static_cast<int32_t>(key_index(best));
    }
    __syncthreads();
    // sibling tokens are distinct, so each slot has at most one matching child
    for (int j = 1 + tid; j < N; j += kNT)
      if (sh.pslot[j] >= 0 && sh.tok[j] == sh.am[sh.pslot[j]]) sh.next[sh.pslot[j]] = j;
    __syncthreads();
    if (tid == 0) {
      int cur = 0, len = 0;
      path_out[0] = 0;
      while (sh.next[cur] >= 0 && len < p.max_depth) {
        cur = sh.next[cur];
        path_out[++len] = cur;
      }
      for (int t = len + 1; t <= p.max_depth; ++t) path_out[t] = -1;
      p.accept_len[b] = len;
      p.bonus[b] = sh.am[cur];
      p.new_ctx[b] = p.ctx[b] + 1 + len;
    }
    return;
  }

  // ---------------------------------------------------------- stochastic
  const T* target = reinterpret_cast<const T*>(p.target);
  const T* draft = reinterpret_cast<const T*>(p.draft);
  const int64_t lo = static_cast<int64_t>(rank) * slice;
  const int64_t hi = min(lo + slice, V);
  int round = 0, cur = 0, len = 0, bonus = -1;
  if (tid == 0) sh.path[0] = 0;
  for (int step = 0; step <= p.max_depth; ++step) {
    const int u = sh.node[cur];
    const float lse_t = row_lse(cur);
    if (tid == 0) {
      int nk = 0;
      for (int j = cur + 1; j < N; ++j)
        if (sh.pslot[j] == cur) sh.kids[nk++] = j;
      sh.n_kids = nk;
    }
    __syncthreads();
    const int nk = sh.n_kids;
    const T* trow = target + (static_cast<int64_t>(b) * p.n_max + cur) * V;
    const T* qrow = nullptr;
    float lse_q = 0.f;
    if (nk > 0) {
      qrow = draft + (static_cast<int64_t>(b) * p.rows_per_seq + p.xrow[nb + u]) * V;
      lse_q = p.xlse[nb + u];
    }
    for (int64_t v = lo + tid; v < hi; v += kNT) {
      ps[v - lo] = __expf(to_f<T>(trow[v]) - lse_t);
      if (nk > 0) qs[v - lo] = __expf(to_f<T>(qrow[v]) - lse_q);
    }
    __syncthreads();
    int accepted = -1, nz = 0;
    const uint64_t pre = hash_prefix(p.seed, b, p.cycle, kStreamRatio, cur);
    for (int c = 0; c < nk; ++c) {
      const int x = sh.tok[sh.kids[c]];
      // p(x) after nz rejections, by the same arithmetic as the slice update
      float px = __expf(to_f<T>(trow[x]) - lse_t);
      const float qx = __expf(to_f<T>(qrow[x]) - lse_q);
      for (int jz = 0; jz < nz; ++jz)
        if (sh.Z[jz] > 0.f) px = fmaxf(px - qx, 0.f) / sh.Z[jz];
      if (uniform_ratio(pre, static_cast<uint64_t>(c)) * qx < px) {
        accepted = sh.kids[c];
        break;
      }
      float part = 0.f;
      for (int64_t v = lo + tid; v < hi; v += kNT) part += fmaxf(ps[v - lo] - qs[v - lo], 0.f);
      part = block_sum<kNT>(part, sh.red);
      const float z = cluster_sum(part, sh.cell_z, round, C);
      if (z > 0.f)
        for (int64_t v = lo + tid; v < hi; v += kNT)
          ps[v - lo] = fmaxf(ps[v - lo] - qs[v - lo], 0.f) / z;
      __syncthreads();
      if (tid == 0) sh.Z[nz] = z;
      ++nz;
      __syncthreads();
    }
    if (accepted >= 0) {
      cur = accepted;
      ++len;
      if (tid == 0 && len <= LTD_MAX_DEPTH) sh.path[len] = cur;
      __syncthreads();
      continue;
    }
    const uint64_t preb = hash_prefix(p.seed, b, p.cycle, kStreamBonus, cur);
    uint64_t bestk = 0ull;
    for (int64_t v = lo + tid; v < hi; v += kNT) {
      const float pv = ps[v - lo];
      if (pv > 0.f) {
        const float g = uniform_gumbel(preb, static_cast<uint64_t>(v));
        const uint64_t key = make_key(logf(pv) - logf(-logf(g)), static_cast<uint32_t>(v));
        bestk = key > bestk ? key : bestk;
      }
    }
    bestk = block_max_u64<kNT>(bestk, sh.redk);
    bestk = cluster_max_u64(bestk, sh.cell_key, round, C);
    bonus = static_cast<int>(key_index(bestk));
    break;
  }
  if (rank == 0 && tid == 0) {
    for (int t = 0; t <= p.max_depth; ++t) path_out[t] = (t <= len) ? sh.path[t] : -1;
    p.accept_len[b] = len;
    p.bonus[b] = bonus;
    p.new_ctx[b] = p.ctx[b] + 1 + len;
  }
  // no CTA leaves while a peer may still read its exchange cells
  tc::cluster_sync();
}

constexpr int kCompactNT = 128;
constexpr int kCompactMaxRowBytes = 512;

__global__ void __launch_bounds__(kCompactNT) kv_compact_kernel(const CompactParams p) {
  __shared__ uint4 buf[(LTD_MAX_DEPTH + 1) * kCompactMaxRowBytes / 16];
  grid_wait();
  trigger_dependents();
  const int h = blockIdx.x, layer = blockIdx.y >> 1, which = blockIdx.y & 1, b = blockIdx.z;
  const int a = p.accept_len[b];
  if (a < 0) return;
  const int ctx = p.ctx[b];
  const int32_t* path = p.path + static_cast<int64_t>(b) * p.path_stride;
  if (a + 1 > p.path_stride || a > LTD_MAX_DEPTH) {
    if (threadIdx.x == 0) flag_error(p.err, LTD_DEVERR_NVERIFY);
    return;
  }
  char* base = static_cast<char*>(which ? p.v_layers[layer] : p.k_layers[layer]) +
               (static_cast<int64_t>(b) * p.hkv + h) * p.s_cap * p.row_bytes;
  const int n16 = p.row_bytes / 16;
  for (int idx = threadIdx.x; idx < (a + 1) * n16; idx += kCompactNT) {
    const int t = idx / n16, w = idx % n16;
    const int src = ctx + path[t];
    if (path[t] < 0 || src >= p.s_cap || ctx + t >= p.s_cap) {
      flag_error(p.err, LTD_DEVERR_CTX);
      continue;
    }
    buf[idx] = reinterpret_cast<const uint4*>(base + static_cast<int64_t>(src) * p.row_bytes)[w];
  }
  __syncthreads();
  for (int idx = threadIdx.x; idx < (a + 1) * n16; idx += kCompactNT) {
    const int t = idx / n16, w = idx % n16;
    const int src = ctx + path[t];
    if (path[t] < 0 || src >= p.s_cap || ctx + t >= p.s_cap || path[t] == t) continue;
    reinterpret_cast<uint4*>(base + static_cast<int64_t>(ctx + t) * p.row_bytes)[w] = buf[idx];
  }
}

}  // namespace

size_t accept_workspace(int32_t batch, int32_t n_max, int64_t vocab) {
  const VocabSplit vs =
      vocab_split(static_cast<int64_t>(batch) * n_max, vocab, kAcceptTargetCtas, kAcceptMinElems);
  const size_t rec = static_cast<size_t>(batch) * n_max * vs.chunks * sizeof(AcceptRecord);
  return (rec + 255) / 256 * 256;
}

template <typename T>
cudaError_t launch_accept_t(const AcceptParams& p, int32_t batch, cudaStream_t s) {
  cudaError_t e = launch(accept_rows_kernel<T>, dim3(p.chunks, p.n_max, batch), dim3(kNT), 0, s,
                         nullptr, 0, p);
  if (e != cudaSuccess) return e;
  // walk cluster: enough CTAs that a vocabulary slice of p and q fits shared memory
  int C = static_cast<int>((p.vocab + 4095) / 4096);
  if (C > 8) C = 8;
  const int need = static_cast<int>((p.vocab + kSliceMax - 1) / kSliceMax);
  if (C < need) C = need;
  if (C < 1) C = 1;
  if (C > kMaxWalkCluster) return cudaErrorInvalidValue;
  const int64_t slice = (p.vocab + C - 1) / C;
  const size_t smem = static_cast<size_t>(2 * slice) * sizeof(float);
  e = cudaFuncSetAttribute(accept_walk_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(accept_walk_kernel<T>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e != cudaSuccess) return e;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  return launch(accept_walk_kernel<T>, dim3(C, batch, 1), dim3(kNT), smem, s, attr, 1, p, C, slice);
}

cudaError_t launch_accept(const AcceptParams& p, int32_t batch, ltd_dtype dtype, cudaStream_t s) {
  return dtype == LTD_BF16 ? launch_accept_t<__nv_bfloat16>(p, batch, s)
                           : launch_accept_t<float>(p, batch, s);
}

cudaError_t launch_compact(const CompactParams& p, int32_t batch, cudaStream_t s) {
  if (p.row_bytes > kCompactMaxRowBytes || p.row_bytes % 16 != 0) return cudaErrorInvalidValue;
  const dim3 grid(p.hkv, p.n_layers * 2, batch);
  return launch(kv_compact_kernel, grid, dim3(kCompactNT), 0, s, nullptr, 0, p);
}

}  // namespace ltd
