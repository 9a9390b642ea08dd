// Acceptance and KV compaction (LTD section 3.2, "Draft Tree Verification").
//
// accept_kernel: grid (chunks, n_max, batch).  Each CTA scans one chunk of
// one verified slot's target row and records (max, sum exp, argmax key).
// The last CTA of a sequence (atomic ticket, no spinning) merges the chunk
// records per slot in a fixed order and walks the verified tree:
//  - greedy: follow the child whose token is the target argmax (ties to the
//    lower token id); the argmax at the first mismatch is the bonus;
//  - stochastic (T = 1): SpecInfer-style multi-candidate speculative
//    sampling -- child i of the current slot is accepted if
//    r_i q(x_i) < p(x_i), else p <- max(p - q, 0) / Z; with no child accepted
//    the bonus is a Gumbel-max draw from p.  The residual p is never stored:
//    every pass re-derives it element-wise from the target row, the draft row
//    and the list of normalisers Z so far.
// kv_compact_kernel: grid (KV heads, layers x {K, V}, batch); each CTA stages
// the accepted rows in shared memory, then writes them to ctx+t, so a row
// that is both a source and a destination is read before it is overwritten.
#include "ltd_common.cuh"
#include "ltd_internal.h"

namespace ltd {

namespace {

constexpr int kNT = 512;

struct WalkShared {
  int32_t node[LTD_MAX_N];
  int32_t tok[LTD_MAX_N];
  int32_t pslot[LTD_MAX_N];
  int32_t am[LTD_MAX_N];
  float lse[LTD_MAX_N];
  int32_t kids[LTD_MAX_N];
  float Z[LTD_MAX_N];
  int32_t path[LTD_MAX_DEPTH + 1];
  int n_kids, next, accepted;
};

// Residual target probability at token v after nz rejections at one node.
template <typename T>
__device__ __forceinline__ float p_chain(const T* trow, const T* qrow, float lp, float lq,
                                         const float* Z, int nz, int64_t v) {
  float pv = __expf(to_f<T>(trow[v]) - lp);
  if (nz > 0) {
    const float qv = __expf(to_f<T>(qrow[v]) - lq);
    for (int j = 0; j < nz; ++j)
      if (Z[j] > 0.f) pv = fmaxf(pv - qv, 0.f) / Z[j];
  }
  return pv;
}

template <typename T>
__device__ void walk(const AcceptParams& p, int b, int N, int mode, WalkShared& sh, float* red,
                     uint64_t* redk) {
  const int tid = threadIdx.x;
  const int64_t nb = static_cast<int64_t>(b) * p.max_nodes;
  const T* target = reinterpret_cast<const T*>(p.target);
  const T* draft = reinterpret_cast<const T*>(p.draft);
  const int64_t V = p.vocab;

  // per-slot merge of the chunk records (fixed order) and tree lookups
  for (int j = tid; j < N; j += kNT) {
    const AcceptRecord* r = p.rec + (static_cast<int64_t>(b) * p.n_max + j) * p.chunks;
    float M = -CUDART_INF_F, S = 0.f;
    unsigned long long best = 0ull;
    for (int c = 0; c < p.chunks; ++c) {
      const float rm = __ldcg(&r[c].m), rs = __ldcg(&r[c].s);
      const unsigned long long rk = __ldcg(&r[c].key);
      ms_merge(M, S, rm, rs);
      best = rk > best ? rk : best;
    }
    sh.am[j] = static_cast<int32_t>(key_index(best));
    sh.lse[j] = M + logf(S);
    const int nid = p.node_ids[static_cast<int64_t>(b) * p.n_max + j];
    sh.node[j] = nid;
    sh.tok[j] = p.token[nb + nid];
  }
  __syncthreads();
  for (int j = tid; j < N; j += kNT) {
    const int par = p.parent[nb + sh.node[j]];
    int lo = 0, hi = j - 1, found = -1;  // slots are ascending node ids
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
  if (tid == 0) sh.path[0] = 0;
  __syncthreads();

  int cur = 0, len = 0, bonus = -1;
  for (int step = 0; step <= p.max_depth; ++step) {
    if (tid == 0) {
      int nk = 0;
      for (int j = cur + 1; j < N; ++j)
        if (sh.pslot[j] == cur) sh.kids[nk++] = j;
      sh.n_kids = nk;
      sh.accepted = -1;
    }
    __syncthreads();
    const int nk = sh.n_kids;
    if (mode == LTD_GREEDY) {
      const int pred = sh.am[cur];
      if (tid == 0)
        for (int c = 0; c < nk; ++c)
          if (sh.tok[sh.kids[c]] == pred) {
            sh.accepted = sh.kids[c];
            break;
          }
      __syncthreads();
      if (sh.accepted < 0) {
        bonus = pred;
        break;
      }
    } else {
      const T* trow = target + (static_cast<int64_t>(b) * p.n_max + cur) * V;
      const float lp = sh.lse[cur];
      const T* qrow = nullptr;
      float lq = 0.f;
      int nz = 0;
      if (nk > 0) {
        const int u = sh.node[cur];
        qrow = draft + (static_cast<int64_t>(b) * p.rows_per_seq + p.xrow[nb + u]) * V;
        lq = p.xlse[nb + u];
        const uint64_t pre = hash_prefix(p.seed, b, p.cycle, kStreamRatio, cur);
        for (int c = 0; c < nk; ++c) {
          if (tid == 0) {
            const int x = sh.tok[sh.kids[c]];
            const float px = p_chain<T>(trow, qrow, lp, lq, sh.Z, nz, x);
            const float qx = __expf(to_f<T>(qrow[x]) - lq);
            const float r = uniform_ratio(pre, static_cast<uint64_t>(c));
            if (r * qx < px) sh.accepted = sh.kids[c];
          }
          __syncthreads();
          if (sh.accepted >= 0) break;
          float part = 0.f;
          for (int64_t v = tid; v < V; v += kNT) {
            const float pv = p_chain<T>(trow, qrow, lp, lq, sh.Z, nz, v);
            const float qv = __expf(to_f<T>(qrow[v]) - lq);
            part += fmaxf(pv - qv, 0.f);
          }
          const float z = block_sum<kNT>(part, red);
          __syncthreads();
          if (tid == 0) sh.Z[nz] = z;
          ++nz;
          __syncthreads();
        }
      }
      if (sh.accepted < 0) {
        const uint64_t pre = hash_prefix(p.seed, b, p.cycle, kStreamBonus, cur);
        uint64_t bestk = 0ull;
        for (int64_t v = tid; v < V; v += kNT) {
          const float pv = p_chain<T>(trow, qrow, lp, lq, sh.Z, nz, v);
          if (pv > 0.f) {
            const float g = uniform_gumbel(pre, static_cast<uint64_t>(v));
            const float sc = logf(pv) - logf(-logf(g));
            const uint64_t key = make_key(sc, static_cast<uint32_t>(v));
            bestk = key > bestk ? key : bestk;
          }
        }
        bestk = block_max_u64<kNT>(bestk, redk);
        bonus = static_cast<int>(key_index(bestk));
        break;
      }
    }
    cur = sh.accepted;
    ++len;
    if (tid == 0) sh.path[len] = cur;
    __syncthreads();
  }
  __syncthreads();
  if (tid == 0) {
    int32_t* path = p.path + static_cast<int64_t>(b) * (p.max_depth + 1);
    for (int t = 0; t <= p.max_depth; ++t) path[t] = (t <= len) ? sh.path[t] : -1;
    p.accept_len[b] = len;
    p.bonus[b] = bonus;
    p.new_ctx[b] = p.ctx[b] + 1 + len;
    p.ticket[b] = 0u;
  }
}

template <typename T>
__global__ void __launch_bounds__(kNT) accept_kernel(const AcceptParams p) {
  constexpr int NW = kNT / kWarp;
  constexpr int VEC = 16 / sizeof(T);
  constexpr int U = 2;
  __shared__ WalkShared sh;
  __shared__ float red[2 * NW];
  __shared__ uint64_t redk[NW];
  __shared__ int s_last;

  const int ch = blockIdx.x, i = blockIdx.y, b = blockIdx.z, tid = threadIdx.x;
  const int N = p.n_verify[b];
  const int mode = p.mode[b];
  if (N < 1 || N > p.n_max || (mode != LTD_GREEDY && mode != LTD_STOCHASTIC)) {
    if (ch == 0 && i == 0 && tid == 0) {
      flag_error(p.err, (N < 1 || N > p.n_max) ? LTD_DEVERR_NVERIFY : LTD_DEVERR_MODE);
      int32_t* path = p.path + static_cast<int64_t>(b) * (p.max_depth + 1);
      for (int t = 0; t <= p.max_depth; ++t) path[t] = -1;
      p.accept_len[b] = -1;
      p.bonus[b] = -1;
      p.new_ctx[b] = p.ctx[b];
    }
    return;
  }
  if (i >= N) return;

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
#pragma unroll
      for (int j = 0; j < VEC; ++j) vm = fmaxf(vm, xv[u][j]);
      if (vm > m) {
        s *= __expf(m - vm);
        m = vm;
      }
#pragma unroll
      for (int j = 0; j < VEC; ++j) {
        if (idx + j < hi) {
          const float xj = xv[u][j];
          s += (xj == -CUDART_INF_F) ? 0.f : __expf(xj - m);
          const uint64_t key = make_key(xj, static_cast<uint32_t>(idx + j));
          best = key > best ? key : best;
        }
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
    __threadfence();
    const uint32_t prev = atomicAdd(&p.ticket[b], 1u);
    s_last = (prev == static_cast<uint32_t>(N * p.chunks - 1));
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  walk<T>(p, b, N, mode, sh, red, redk);
}

constexpr int kCompactNT = 128;
constexpr int kCompactMaxRowBytes = 512;

__global__ void __launch_bounds__(kCompactNT) kv_compact_kernel(const CompactParams p) {
  __shared__ uint4 buf[(LTD_MAX_DEPTH + 1) * kCompactMaxRowBytes / 16];
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
  return (rec + 255) / 256 * 256 + (static_cast<size_t>(batch) * sizeof(uint32_t) + 255) / 256 * 256;
}

cudaError_t launch_accept(const AcceptParams& p, int32_t batch, ltd_dtype dtype, cudaStream_t s) {
  const dim3 grid(p.chunks, p.n_max, batch);
  if (dtype == LTD_BF16) accept_kernel<__nv_bfloat16><<<grid, kNT, 0, s>>>(p);
  else accept_kernel<float><<<grid, kNT, 0, s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_compact(const CompactParams& p, int32_t batch, cudaStream_t s) {
  if (p.row_bytes > kCompactMaxRowBytes || p.row_bytes % 16 != 0) return cudaErrorInvalidValue;
  const dim3 grid(p.hkv, p.n_layers * 2, batch);
  kv_compact_kernel<<<grid, kCompactNT, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace ltd
