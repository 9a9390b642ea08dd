// Acceptance and KV compaction (LTD section 3.2, "Draft Tree Verification").
//
// accept_rows_kernel: every 16 KB unit of every verified slot's target row
// gets (max m, sum exp((x - m) / T), argmax key) in the workspace, one
// 256-thread CTA per unit.
// accept_walk_kernel: one thread-block cluster of C CTAs per sequence.
//  - greedy: rank 0 merges the argmax records (ties to the lower token id),
//    marks every slot whose token is its parent's argmax, and follows those
//    marks from slot 0; the argmax at the end is the bonus token;
//  - stochastic: SpecInfer-style multi-candidate speculative sampling at a
//    temperature T (p and q the softmax of the rows divided by T; at T != 1
//    the draft row's normaliser is reduced over the cluster, at T = 1 the
//    expansion's is used).  Each CTA holds one vocabulary slice of p (target) and q
//    (draft) in its threads' registers.  Child i of the current slot is accepted if
//    r_i q(x_i) < p(x_i) -- every CTA evaluates that test identically --
//    else p <- max(p - q, 0) / Z, with Z summed over the cluster through
//    distributed shared memory (every warp adds all warp partials of the
//    cluster in one fixed order, so every CTA holds the same Z).  The
//    children's p(x), q(x) are loaded with the slice; a rejection costs one
//    cluster barrier and one pass over the slice, which also takes the next
//    rejection's partial sum.  With no child accepted the bonus is a Gumbel-max
//    draw from p, reduced over the cluster the same way;
//  - stochastic with point-mass proposals: child i is accepted if
//    r_i (1 - p(rejected so far)) < p(x_i), with p(x_i) loaded with the
//    slice as above; a rejection only adds p(x_i) to the removed mass (no
//    pass, no barrier), and the Gumbel-max bonus skips the rejected tokens;
//  - stochastic for children drawn from q without replacement: as the first
//    stochastic rule, but after a rejection the rejected token's q is zeroed
//    (in its owner thread's registers) and q renormalised by a scalar,
//    1 / (1 - q-mass of the rejected children), in the same pass as the
//    residual update.
// kv_append_kernel: the verified tokens' new K/V rows into every layer's cache.
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
static_assert(LTD_MAX_N <= kNT, "one verified slot per walk thread");

// 2^x by the hardware's approximate base-2 exponential (ex2.approx.ftz).
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

constexpr int kRowUnitBytes = 16384;  // one unit: 16 KB of one verified row
constexpr int kRowNT = 256;            // one CTA per unit
constexpr int kRowNW = kRowNT / kWarp;
constexpr int kRowVecs = kRowUnitBytes / 16 / kRowNT;  // 16-byte vectors per thread

// Row statistics of the verified slots' target rows: every unit (16 KB of
// one row) gets (max m, sum exp((x - m) / T), argmax key) in the workspace,
// one CTA per unit.  Each thread's four loads are in flight before the first
// is used; the warps' partials meet in shared memory after one barrier.
template <typename T>
__global__ void __launch_bounds__(kRowNT, 8) accept_rows_kernel(const AcceptParams p) {
  constexpr int VEC = 16 / sizeof(T);
  __shared__ float pm[kRowNW], ps[kRowNW];
  __shared__ uint64_t pk[kRowNW];
  grid_wait();
  trigger_dependents();
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int u = static_cast<int>(blockIdx.x);
  const int c = u % p.chunks, bi = u / p.chunks;
  const int i = bi % p.n_max, b = bi / p.n_max;
  const int N = __ldcg(p.n_verify + b);
  const int mode = __ldcg(p.mode + b);
  if (N < 1 || N > p.n_max || i >= N) return;  // (the walk flags a bad N)
  const int lo = c * static_cast<int>(p.chunk_elems);
  const int n_here = min(static_cast<int>(p.chunk_elems), static_cast<int>(p.vocab) - lo);
  const T* row = reinterpret_cast<const T*>(p.target) + (static_cast<int64_t>(b) * p.n_max + i) * p.vocab + lo;
  uint4 v[kRowVecs];
#pragma unroll
  for (int k = 0; k < kRowVecs; ++k) {
    const int e = (k * kRowNT + tid) * VEC;  // rows end on a 16-byte boundary
    v[k] = (e < n_here) ? ld_stream16_once(row + e)
                        : ((sizeof(T) == 4) ? make_uint4(0xFF800000u, 0xFF800000u, 0xFF800000u, 0xFF800000u)
                                            : make_uint4(0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u));
  }
  // the thread's max (the first, so the lowest token) and -- for the
  // stochastic rules only: greedy needs no normaliser -- its sum of
  // 2^((x - max) c), c = log2(e) / T, one vector at a time (the sum
  // rescaled when the max grows)
  const bool stoch = mode != LTD_GREEDY;
  const float cl = p.inv_t * 1.4426950408889634f;
  float tm = -CUDART_INF_F, ts = 0.f;
  int ti = 0;
#pragma unroll
  for (int k = 0; k < kRowVecs; ++k) {
    float vm = -CUDART_INF_F;
    int jm = 0;
#pragma unroll
    for (int j = 0; j < VEC; ++j) {
      const float x = elem<T>(v[k], j);
      if (x > vm) {
        vm = x;
        jm = j;
      }
    }
    if (vm > tm) {
      ts = (stoch && tm > -CUDART_INF_F) ? ts * ex2_approx((tm - vm) * cl) : 0.f;
      tm = vm;
      ti = (k * kRowNT + tid) * VEC + jm;
    }
    if (stoch && tm > -CUDART_INF_F) {
      const float off = -tm * cl;
#pragma unroll
      for (int j = 0; j < VEC; ++j) ts += ex2_approx(fmaf(elem<T>(v[k], j), cl, off));
    }
  }
  // warp, then CTA: the max first, then each sum rescaled to it
  float M = tm;
  uint64_t K = (tm > -CUDART_INF_F) ? make_key(tm, static_cast<uint32_t>(lo + ti)) : 0ull;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    M = fmaxf(M, __shfl_xor_sync(0xFFFFFFFFu, M, o));
    const uint64_t ok = __shfl_xor_sync(0xFFFFFFFFu, K, o);
    K = ok > K ? ok : K;
  }
  float e = (tm > -CUDART_INF_F) ? ts * __expf((tm - M) * p.inv_t) : 0.f;
  e = warp_sum_f(e);
  if (lane == 0) {
    pm[warp] = M;
    ps[warp] = e;
    pk[warp] = K;
  }
  __syncthreads();
  if (warp == 0) {
    float wm = lane < kRowNW ? pm[lane] : -CUDART_INF_F;
    float we = lane < kRowNW ? ps[lane] : 0.f;
    uint64_t wk = lane < kRowNW ? pk[lane] : 0ull;
    float MM = wm;
#pragma unroll
    for (int o = kRowNW / 2; o > 0; o >>= 1) {
      MM = fmaxf(MM, __shfl_xor_sync(0xFFFFFFFFu, MM, o));
      const uint64_t ok = __shfl_xor_sync(0xFFFFFFFFu, wk, o);
      wk = ok > wk ? ok : wk;
    }
    float se = (wm > -CUDART_INF_F) ? we * __expf((wm - MM) * p.inv_t) : 0.f;
#pragma unroll
    for (int o = kRowNW / 2; o > 0; o >>= 1) se += __shfl_xor_sync(0xFFFFFFFFu, se, o);
    if (lane == 0) {
      AcceptRecord* r = p.rec + static_cast<int64_t>(u);  // [batch][n_max][chunks] = unit order
      r->m = MM;
      r->s = se;
      r->key = wk;
    }
  }
}

// Optional walk timeline for performance work (off in normal builds):
// per sequence, (event, globaltimer) pairs from rank 0's thread 0.
#ifdef LTD_TRACE
__device__ unsigned long long g_walk_trace[64][128];
__device__ int g_walk_trace_n[64];
#define WTRACE(ev)                                                              \
  do {                                                                          \
    if (rank == 0 && tid == 0 && b < 64) {                                      \
      const int i_ = g_walk_trace_n[b];                                         \
      if (i_ < 64) {                                                            \
        g_walk_trace[b][2 * i_] = (ev);                                         \
        g_walk_trace[b][2 * i_ + 1] = tc::globaltimer();                        \
        g_walk_trace_n[b] = i_ + 1;                                             \
      }                                                                         \
    }                                                                           \
  } while (0)
#else
#define WTRACE(ev) \
  do {             \
  } while (0)
#endif

struct WalkShared {
  int32_t node[LTD_MAX_N];
  int32_t tok[LTD_MAX_N];
  int32_t pslot[LTD_MAX_N];
  int32_t am[LTD_MAX_N];
  int32_t next[LTD_MAX_N];
  int32_t kids[LTD_MAX_N];
  float Z[LTD_MAX_N];
  float S[LTD_MAX_N];  // without-replacement rule: scale of q at each rejection
  int32_t path[LTD_MAX_DEPTH + 1];
  float red[2 * kNW];
  uint64_t redk[kNW];
  unsigned long long bestk[LTD_MAX_N];  // greedy: each slot's argmax key
  float kp[LTD_MAX_N];      // p and q of the current slot's children
  float kq[LTD_MAX_N];
  float wpart[2][kMaxWalkCluster][kNW];  // every CTA's warp sums, by round parity
  int wcnt[kNW];
  uint64_t cell_key[2];
  float2 cell_ms;
  int n_kids;
};

// Sum over the cluster of every thread's `v`: every warp pushes its sum into
// every CTA's table ([round parity][rank][warp]) before the cluster barrier,
// then every warp adds its own CTA's table in one fixed order, so every
// thread of every CTA holds the same bits.  One cluster barrier, no remote
// reads after it.
__device__ __forceinline__ float cluster_sum_warps(float v, float (*wpart)[kMaxWalkCluster][kNW],
                                                  int& round, int C) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int c = round & 1;
  const uint32_t rank = tc::cluster_rank();
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
  if (lane < C) tc::st_cluster_f1(tc::mapa(tc::smem_u32(&wpart[c][rank][warp]), lane), v);
  tc::cluster_sync();
  float t = 0.f;
  for (int e = lane; e < C * kNW; e += kWarp) t += wpart[c][e / kNW][e % kNW];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xFFFFFFFFu, t, o);
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
                                                          int64_t slice, int vec_ok) {
  __shared__ WalkShared sh;
  for (int j = threadIdx.x; j < LTD_MAX_N; j += kNT) sh.bestk[j] = 0ull;
  __syncthreads();
  grid_wait();
  trigger_dependents();
  const int rank = blockIdx.x, b = blockIdx.y, tid = threadIdx.x;
  // the sequence's scalars and its slots' node ids are fetched together
  // (the node ids do not depend on N; one slot per thread, n_max <= kNT)
  const int N = __ldcg(p.n_verify + b);
  const int mode = __ldcg(p.mode + b);
  const int nid_pre = (tid < p.n_max) ? __ldcg(p.node_ids + static_cast<int64_t>(b) * p.n_max + tid) : 0;
  int32_t* path_out = p.path + static_cast<int64_t>(b) * (p.max_depth + 1);
  // everything below is uniform over the cluster (one sequence)
  if (N < 1 || N > p.n_max ||
      (mode != LTD_GREEDY && mode != LTD_STOCHASTIC && mode != LTD_STOCHASTIC_POINT_MASS &&
       mode != LTD_STOCHASTIC_NO_REPLACEMENT)) {
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
  if (mode == LTD_GREEDY) {
    // every slot's argmax over its row's units: one pass over the records
    // (all loads independent), max-combined in shared memory
    const AcceptRecord* r0 = p.rec + static_cast<int64_t>(b) * p.n_max * p.chunks;
    for (int r = tid; r < N * p.chunks; r += kNT) atomicMax(&sh.bestk[r / p.chunks], r0[r].key);
  }
  // each slot's token and parent node (both loads in flight together)
  if (tid < N) {
    sh.node[tid] = nid_pre;
    sh.tok[tid] = p.token[nb + nid_pre];
    sh.pslot[tid] = p.parent[nb + nid_pre];  // the parent's node id for now
    sh.next[tid] = -1;
  }
  __syncthreads();
  if (tid < N) {
    const int par = sh.pslot[tid];
    int lo = 0, hi = tid - 1, found = -1;  // slots hold ascending node ids
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
    sh.pslot[tid] = found;  // (only this thread reads its entry)
  }
  __syncthreads();
  // log-sum-exp of the target row at slot over the vocabulary, in units of
  // logit / T: the chunks' (max, sum exp((x - max) / T)) merged
  auto row_lse = [&](int slot) {
    const AcceptRecord* r = p.rec + (static_cast<int64_t>(b) * p.n_max + slot) * p.chunks;
    float M = -CUDART_INF_F, S = 0.f;
    for (int c = 0; c < p.chunks; ++c) {
      const float m2 = r[c].m, s2 = r[c].s;
      if (m2 == -CUDART_INF_F) continue;
      if (M == -CUDART_INF_F) {
        M = m2;
        S = s2;
        continue;
      }
      const float mm = fmaxf(M, m2);
      S = S * __expf((M - mm) * p.inv_t) + s2 * __expf((m2 - mm) * p.inv_t);
      M = mm;
    }
    return M * p.inv_t + logf(S);
  };

  if (mode == LTD_GREEDY) {
    for (int j = tid; j < N; j += kNT) sh.am[j] = static_cast<int32_t>(key_index(sh.bestk[j]));
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
  const bool pm = mode == LTD_STOCHASTIC_POINT_MASS;     // no q: children are point masses
  const bool nr = mode == LTD_STOCHASTIC_NO_REPLACEMENT;  // q loses each rejected child
  const T* target = reinterpret_cast<const T*>(p.target);
  const T* draft = reinterpret_cast<const T*>(p.draft);
  const int64_t lo = static_cast<int64_t>(rank) * slice;
  const int64_t hi = min(lo + slice, V);
  // The slice lives in registers: KG groups of VEC elements per thread.
  // With 16-byte-aligned rows (vec_ok) group k of a thread is the VEC
  // consecutive elements at lo + (k kNT + tid) VEC, loaded with one 16-byte
  // load; otherwise element (k, j) is lo + (k VEC + j) kNT + tid.
  constexpr int VEC = 16 / static_cast<int>(sizeof(T));
  constexpr int KG = static_cast<int>(kSliceMax) / (VEC * kNT);
  static_assert(KG * VEC * kNT == kSliceMax, "slices split evenly over the threads");
  auto el = [&](int k, int j) -> int64_t {
    return vec_ok ? lo + (static_cast<int64_t>(k) * kNT + tid) * VEC + j
                  : lo + (static_cast<int64_t>(k) * VEC + j) * kNT + tid;
  };
  float pr[KG][VEC], qr[KG][VEC];
  int round = 0, cur = 0, len = 0, bonus = -1;
  if (tid == 0) sh.path[0] = 0;
  const int lane = tid & 31, warp = tid >> 5;
  WTRACE(0);
  for (int step = 0; step <= p.max_depth; ++step) {
    const int u = sh.node[cur];
    const float lse_t = row_lse(cur);
    WTRACE(1);
    // the current slot's children, in slot order (one slot per thread)
    {
      const bool kid = tid < N && tid > cur && sh.pslot[tid] == cur;
      const unsigned bal = __ballot_sync(0xFFFFFFFFu, kid);
      if (lane == 0) sh.wcnt[warp] = __popc(bal);
      __syncthreads();
      int before = 0, total = 0;
      for (int w = 0; w < kNW; ++w) {
        before += (w < warp) ? sh.wcnt[w] : 0;
        total += sh.wcnt[w];
      }
      if (kid) sh.kids[before + __popc(bal & ((1u << lane) - 1u))] = tid;
      if (tid == 0) sh.n_kids = total;
    }
    __syncthreads();
    const int nk = sh.n_kids;
    WTRACE(2 + 100 * nk);
    const T* trow = target + (static_cast<int64_t>(b) * p.n_max + cur) * V;
    const T* qrow = nullptr;
    float lse_q = 0.f;
    const bool use_q = nk > 0 && !pm;
    if (use_q) {
      qrow = draft + (static_cast<int64_t>(b) * p.rows_per_seq + p.xrow[nb + u]) * V;
      lse_q = p.xlse[nb + u];
    }
    const float it = p.inv_t;
    // the children's p(x) and this CTA's slice, all loads at once; the slice
    // pass also takes this thread's share of the first residual sum.  The
    // slice goes 16 bytes of logits per thread-step where the rows allow it
    // (groups of VEC elements), the rest one element at a time.
    if (tid < nk) sh.kp[tid] = __expf(to_f<T>(trow[sh.tok[sh.kids[tid]]]) * it - lse_t);
    float part = 0.f;
    {
      uint4 rt[KG], rq[KG];
#pragma unroll
      for (int k = 0; k < KG; ++k) {
        // every load of the slice is issued before the first is used
        rt[k] = make_uint4(0u, 0u, 0u, 0u);
        rq[k] = make_uint4(0u, 0u, 0u, 0u);
        if (vec_ok && el(k, 0) < hi) {
          rt[k] = ld_stream16_once(trow + el(k, 0));
          if (use_q) rq[k] = ld_stream16_once(qrow + el(k, 0));
        }
      }
      auto dval = [&](int k, int j) -> float {
        return vec_ok ? elem<T>(rq[k], j) : to_f<T>(qrow[el(k, j)]);
      };
      if (use_q && p.tempered) {
        // q = softmax(draft row / T): its log-sum-exp over the vocabulary,
        // the cluster's max of the row, then the cluster's sum of
        // exp((x - max) / T)
        float tm = -CUDART_INF_F;
#pragma unroll
        for (int k = 0; k < KG; ++k)
#pragma unroll
          for (int j = 0; j < VEC; ++j)
            if (el(k, j) < hi) tm = fmaxf(tm, dval(k, j));
        uint64_t km = block_max_u64<kNT>(make_key(tm, 0u), sh.redk);
        km = cluster_max_u64(km, sh.cell_key, round, C);
        const float qm = key_value(km);
        float ts = 0.f;
#pragma unroll
        for (int k = 0; k < KG; ++k)
#pragma unroll
          for (int j = 0; j < VEC; ++j)
            if (el(k, j) < hi) ts += __expf((dval(k, j) - qm) * it);
        lse_q = qm * it + logf(cluster_sum_warps(ts, sh.wpart, round, C));
      }
      if (tid < nk) sh.kq[tid] = use_q ? __expf(to_f<T>(qrow[sh.tok[sh.kids[tid]]]) * it - lse_q) : 0.f;
#pragma unroll
      for (int k = 0; k < KG; ++k)
#pragma unroll
        for (int j = 0; j < VEC; ++j) {
          const int64_t v = el(k, j);
          const bool in = v < hi;
          float tv = 0.f, dv = 0.f;
          if (vec_ok) {
            tv = elem<T>(rt[k], j);
            dv = elem<T>(rq[k], j);
          } else if (in) {
            tv = to_f<T>(trow[v]);
            if (use_q) dv = to_f<T>(qrow[v]);
          }
          pr[k][j] = 0.f;
          qr[k][j] = 0.f;
          if (in) {
            pr[k][j] = __expf(tv * it - lse_t);
            if (use_q) qr[k][j] = __expf(dv * it - lse_q);
          }
          part += fmaxf(pr[k][j] - qr[k][j], 0.f);
        }
    }
    __syncthreads();
    WTRACE(3);
    int accepted = -1, nz = 0;
    const uint64_t pre = hash_prefix(p.seed, b, p.cycle, kStreamRatio, cur);
    float removed = 0.f;  // point-mass rule: p mass of the rejected children
    float qs = 1.f, qrej = 0.f;  // without replacement: q scale, q mass rejected
    for (int c = 0; c < nk; ++c) {
      if (pm) {
        const float px = sh.kp[c];
        if (uniform_ratio(pre, static_cast<uint64_t>(c)) * (1.f - removed) < px) {
          accepted = sh.kids[c];
          break;
        }
        removed += px;
        ++nz;
        continue;
      }
      // p(x) after nz rejections, by the same arithmetic as the slice update
      // (sh.Z holds 1 / Z, or 0 where the residual was empty; sh.S the scale
      // of q at that rejection, 1 unless q loses its rejected children)
      float px = sh.kp[c];
      const float qx = sh.kq[c];
      for (int jz = 0; jz < nz; ++jz)
        if (sh.Z[jz] > 0.f) px = fmaxf(px - qx * sh.S[jz], 0.f) * sh.Z[jz];
      if (uniform_ratio(pre, static_cast<uint64_t>(c)) * (qx * qs) < px) {
        accepted = sh.kids[c];
        break;
      }
      const float z = cluster_sum_warps(part, sh.wpart, round, C);
      WTRACE(4);
      const float zi = z > 0.f ? __frcp_rn(z) : 0.f;
      // without replacement: the rejected token leaves q, the rest rescales
      const int64_t xrej = nr ? static_cast<int64_t>(sh.tok[sh.kids[c]]) : -1;
      float qs_next = qs;
      if (nr) {
        qrej += qx;
        qs_next = (1.f - qrej) > 0.f ? __frcp_rn(1.f - qrej) : 0.f;
      }
      // the residual update, with this thread's share of the next sum (the
      // plain rule keeps q as it is: its own loop, without the q scaling)
      part = 0.f;
      if (nr) {
#pragma unroll
        for (int k = 0; k < KG; ++k)
#pragma unroll
          for (int j = 0; j < VEC; ++j) {
            if (zi > 0.f) pr[k][j] = fmaxf(pr[k][j] - qr[k][j] * qs, 0.f) * zi;
            if (el(k, j) == xrej) qr[k][j] = 0.f;
            part += fmaxf(pr[k][j] - qr[k][j] * qs_next, 0.f);
          }
      } else {
#pragma unroll
        for (int k = 0; k < KG; ++k)
#pragma unroll
          for (int j = 0; j < VEC; ++j) {
            if (zi > 0.f) pr[k][j] = fmaxf(pr[k][j] - qr[k][j], 0.f) * zi;
            part += fmaxf(pr[k][j] - qr[k][j], 0.f);
          }
      }
      // every thread records the same values, so no barrier is needed before
      // any thread reads them back
      sh.Z[nz] = zi;
      sh.S[nz] = qs;
      qs = qs_next;
      ++nz;
      WTRACE(5);
    }
    if (accepted >= 0) {
      cur = accepted;
      ++len;
      if (tid == 0 && len <= LTD_MAX_DEPTH) sh.path[len] = cur;
      __syncthreads();
      continue;
    }
    const uint64_t preb = hash_prefix(p.seed, b, p.cycle, kStreamBonus, cur);
    // Gumbel-max: the largest log p(v) + G_v, with G_v = -log(-log u_v),
    // ranked as p(v) / (-log u_v) (the same order)
    uint64_t bestk = 0ull;
    // the point-mass rule draws the bonus from p without the rejected children
    auto rejected = [&](int64_t v) {
      bool r = false;
      if (pm)
        for (int c = 0; c < nz; ++c) r |= sh.tok[sh.kids[c]] == static_cast<int32_t>(v);
      return r;
    };
    auto offer = [&](float pv, int64_t v) {
      if (pv > 0.f && !rejected(v)) {
        const float e = -__logf(uniform_gumbel(preb, static_cast<uint64_t>(v)));
        const uint64_t key = make_key(__fdividef(pv, e), static_cast<uint32_t>(v));
        bestk = key > bestk ? key : bestk;
      }
    };
    // (a loop the size of one group, run KG times: this code runs once per
    // sequence, so its instruction fetch, not its arithmetic, would dominate
    // if it were unrolled over the whole slice)
#pragma unroll 1
    for (int k = 0; k < KG; ++k) {
      if (el(k, 0) >= hi) continue;
      float pk[VEC];
#pragma unroll
      for (int j = 0; j < VEC; ++j) {
        float x = pr[0][j];
#pragma unroll
        for (int kk = 1; kk < KG; ++kk) x = (k == kk) ? pr[kk][j] : x;
        pk[j] = x;
      }
#pragma unroll
      for (int j = 0; j < VEC; ++j)
        if (el(k, j) < hi) offer(pk[j], el(k, j));
    }
    WTRACE(8);
    bestk = block_max_u64<kNT>(bestk, sh.redk);
    WTRACE(9);
    bestk = cluster_max_u64(bestk, sh.cell_key, round, C);
    bonus = static_cast<int>(key_index(bestk));
    WTRACE(6);
    break;
  }
  WTRACE(7);
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

// Grid (hkv, layers x {K, V}, batch): one CTA copies one head's N new rows
// (whole 16-byte units, coalesced) to rows ctx .. ctx + N - 1.
__global__ void __launch_bounds__(kCompactNT) kv_append_kernel(const AppendParams p) {
  grid_wait();
  trigger_dependents();
  const int h = blockIdx.x, layer = blockIdx.y >> 1, which = blockIdx.y & 1, b = blockIdx.z;
  const int ctx = p.ctx[b], N = p.n_verify[b];
  if (N < 1 || N > p.n_max || ctx < 0 || ctx + N > p.s_cap) {
    if (threadIdx.x == 0 && h == 0 && blockIdx.y == 0)
      flag_error(p.err, (N < 1 || N > p.n_max) ? LTD_DEVERR_NVERIFY : LTD_DEVERR_CTX);
    return;
  }
  const int64_t head = (static_cast<int64_t>(layer) * p.batch + b) * p.hkv + h;
  const uint4* src = reinterpret_cast<const uint4*>((which ? p.new_v : p.new_k) +
                                                    head * p.n_max * p.row_bytes);
  uint4* dst = reinterpret_cast<uint4*>(static_cast<char*>(which ? p.v_layers[layer]
                                                                 : p.k_layers[layer]) +
                                        ((static_cast<int64_t>(b) * p.hkv + h) * p.s_cap + ctx) *
                                            p.row_bytes);
  const int n = N * (p.row_bytes / 16);
  for (int i = threadIdx.x; i < n; i += kCompactNT) dst[i] = __ldcs(src + i);
}

}  // namespace

cudaError_t launch_append(const AppendParams& p, cudaStream_t s) {
  if (p.row_bytes % 16 != 0) return cudaErrorInvalidValue;
  const dim3 grid(p.hkv, p.n_layers * 2, p.batch);
  return launch(kv_append_kernel, grid, dim3(kCompactNT), 0, s, nullptr, 0, p);
}

// One record per row unit, sized for the smaller (fp32) unit.
size_t accept_workspace(int32_t batch, int32_t n_max, int64_t vocab) {
  const int64_t unit = kRowUnitBytes / 4;
  const size_t rec = static_cast<size_t>(batch) * n_max * ((vocab + unit - 1) / unit) * sizeof(AcceptRecord);
  return (rec + 255) / 256 * 256;
}

template <typename T>
cudaError_t launch_accept_t(const AcceptParams& params, int32_t batch, cudaStream_t s) {
  AcceptParams p = params;
  p.chunk_elems = kRowUnitBytes / static_cast<int>(sizeof(T));
  p.chunks = static_cast<int32_t>((p.vocab + p.chunk_elems - 1) / p.chunk_elems);
  const int64_t units = static_cast<int64_t>(batch) * p.n_max * p.chunks;
  if (units > 0x7FFFFFFF) return cudaErrorInvalidValue;
  p.n_units = static_cast<int32_t>(units);
  cudaError_t e = launch(accept_rows_kernel<T>, dim3(static_cast<unsigned>(units)), dim3(kRowNT), 0, s, nullptr,
                         0, p);
  if (e != cudaSuccess) return e;
  // walk cluster: enough CTAs that a vocabulary slice of p and q fits the
  // threads' registers (kSliceMax elements per CTA)
  int C = static_cast<int>((p.vocab + 4095) / 4096);
  if (C > 8) C = 8;
  const int need = static_cast<int>((p.vocab + kSliceMax - 1) / kSliceMax);
  if (C < need) C = need;
  if (C < 1) C = 1;
  if (C > kMaxWalkCluster) return cudaErrorInvalidValue;
  const int64_t slice = ((p.vocab + C - 1) / C + 7) / 8 * 8;  // whole 16-byte groups
  constexpr int kVec = 16 / static_cast<int>(sizeof(T));
  const int vec_ok = (p.vocab % kVec == 0) && (reinterpret_cast<uintptr_t>(p.target) % 16 == 0) &&
                     (reinterpret_cast<uintptr_t>(p.draft) % 16 == 0);
  e = cudaFuncSetAttribute(accept_walk_kernel<T>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e != cudaSuccess) return e;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  return launch(accept_walk_kernel<T>, dim3(C, batch, 1), dim3(kNT), 0, s, attr, 1, p, C, slice,
                vec_ok);
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

#ifdef LTD_TRACE
extern "C" int ltd_walk_trace_read(unsigned long long* host, int* counts) {
  if (cudaMemcpyFromSymbol(host, g_walk_trace, sizeof(g_walk_trace)) != cudaSuccess) return 1;
  return cudaMemcpyFromSymbol(counts, g_walk_trace_n, sizeof(g_walk_trace_n)) == cudaSuccess ? 0 : 1;
}
extern "C" int ltd_walk_trace_clear() {
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_walk_trace_n) != cudaSuccess) return 1;
  return cudaMemset(p, 0, sizeof(g_walk_trace_n)) == cudaSuccess ? 0 : 1;
}
#endif

}  // namespace ltd
