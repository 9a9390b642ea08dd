// Candidate token selection (LTD section 3.2, "Candidate Token Selection").
//
// One CTA per sequence.  Every node gets the key (cum desc, id asc) in
// shared memory (the root gets the maximum key, so it always ranks first);
// one warp per node counts how many keys beat it -- a node is verified iff
// that rank is below N.  A block-wide exclusive scan over the
// flags in id order gives each verified node its slot, so slots are the
// verified ids in ascending order.  Each slot then walks its parent chain
// (at most max_depth steps) and sets one mask bit per ancestor.  Because a
// child's cum never exceeds its parent's and parents have smaller ids, the
// verified set is ancestor-closed; a violation is flagged, not trapped.
#include "ltd_common.cuh"
#include "ltd_internal.h"

namespace ltd {

namespace {

constexpr int kNT = 1024;

__global__ void __launch_bounds__(kNT) select_kernel(const SelectParams p) {
  extern __shared__ __align__(16) unsigned char smem[];
  const int W32 = (p.n_max + 31) / 32;
  uint64_t* keys = reinterpret_cast<uint64_t*>(smem);                          // [max_nodes]
  int32_t* slot_of = reinterpret_cast<int32_t*>(keys + p.max_nodes);          // [max_nodes]
  int32_t* par_s = slot_of + p.max_nodes;                                     // [max_nodes]
  uint32_t* words = reinterpret_cast<uint32_t*>(par_s + p.max_nodes);         // [n_max][W32]
  __shared__ int32_t warp_tot[kNT / kWarp];

  grid_wait();
  trigger_dependents();
  const int b = blockIdx.x, tid = threadIdx.x;
  const int64_t nb = static_cast<int64_t>(b) * p.max_nodes;
  const int n = p.n_nodes[b];
  const int N = p.n_verify[b];
  const int ctx = p.ctx[b];
  int32_t* ids_out = p.node_ids + static_cast<int64_t>(b) * p.n_max;
  int32_t* pos_out = p.pos + static_cast<int64_t>(b) * p.n_max;
  uint32_t* mask_out = p.mask + static_cast<int64_t>(b) * p.n_max * W32;

  const bool ok = (n >= 1 && n <= p.max_nodes && N >= 1 && N <= n && N <= p.n_max);
  if (!ok) {
    if (tid == 0) flag_error(p.err, LTD_DEVERR_NVERIFY);
    for (int i = tid; i < p.n_max; i += kNT) {
      ids_out[i] = -1;
      pos_out[i] = -1;
    }
    for (int i = tid; i < p.n_max * W32; i += kNT) mask_out[i] = 0u;
    return;
  }

  for (int i = tid; i < n; i += kNT) {
    keys[i] = (i == 0) ? ~0ull : make_key(p.cum[nb + i], static_cast<uint32_t>(i));
    par_s[i] = p.parent[nb + i];
  }
  for (int i = tid; i < p.n_max * W32; i += kNT) words[i] = 0u;
  __syncthreads();

  // rank = number of keys strictly greater; verified iff rank < N.  One warp
  // per node, its lanes splitting the key scan; the flag lands in slot_of.
  const int lane = tid & 31, warp = tid >> 5;
  for (int i = warp; i < n; i += kNT / kWarp) {
    const uint64_t ki = keys[i];
    int cnt = 0;
    for (int j = lane; j < n; j += kWarp) cnt += (keys[j] > ki) ? 1 : 0;
    cnt = __reduce_add_sync(0xFFFFFFFFu, cnt);
    if (lane == 0) slot_of[i] = (cnt < N) ? 1 : 0;
  }
  __syncthreads();
  // each thread owns ids [4 tid, 4 tid + 4) so the scan below is in id order
  constexpr int PER = 4;
  int flags[PER];
  int local = 0;
#pragma unroll
  for (int r = 0; r < PER; ++r) {
    const int i = tid * PER + r;
    flags[r] = (i < n) ? slot_of[i] : 0;
    local += flags[r];
  }
  __syncthreads();
  // block exclusive scan of `local`
  int incl = local;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
    if (lane >= o) incl += y;
  }
  if (lane == 31) warp_tot[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    int w = (lane < kNT / kWarp) ? warp_tot[lane] : 0;
    int wi = w;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xFFFFFFFFu, wi, o);
      if (lane >= o) wi += y;
    }
    if (lane < kNT / kWarp) warp_tot[lane] = wi - w;  // exclusive warp offsets
  }
  __syncthreads();
  int slot = warp_tot[warp] + incl - local;
#pragma unroll
  for (int r = 0; r < PER; ++r) {
    const int i = tid * PER + r;
    if (i < n) {
      slot_of[i] = flags[r] ? slot : -1;
      if (flags[r]) {
        ids_out[slot] = i;
        pos_out[slot] = ctx + p.depth[nb + i];
        ++slot;
      }
    }
  }
  __syncthreads();

  // ancestor bits: the thread owning node i writes row slot_of[i] alone
  for (int i = tid; i < n; i += kNT) {
    const int si = slot_of[i];
    if (si < 0) continue;
    uint32_t* row = words + si * W32;
    int a = i;
    int guard = 0;
    while (a >= 0 && guard <= LTD_MAX_DEPTH + 1) {
      const int sa = slot_of[a];
      if (sa < 0) {
        flag_error(p.err, LTD_DEVERR_TREE);
        break;
      }
      row[sa >> 5] |= 1u << (sa & 31);
      a = par_s[a];
      ++guard;
    }
  }
  __syncthreads();
  for (int i = tid; i < p.n_max * W32; i += kNT) mask_out[i] = (i < N * W32) ? words[i] : 0u;
  for (int i = N + tid; i < p.n_max; i += kNT) {
    ids_out[i] = -1;
    pos_out[i] = -1;
  }
}

}  // namespace

cudaError_t launch_select(const SelectParams& p, int32_t batch, cudaStream_t s) {
  const int W32 = (p.n_max + 31) / 32;
  const size_t smem = static_cast<size_t>(p.max_nodes) * (sizeof(uint64_t) + 2 * sizeof(int32_t)) +
                      static_cast<size_t>(p.n_max) * W32 * sizeof(uint32_t);
  cudaError_t e = cudaFuncSetAttribute(select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  return launch(select_kernel, dim3(batch), dim3(kNT), smem, s, nullptr, 0, p);
}

}  // namespace ltd
