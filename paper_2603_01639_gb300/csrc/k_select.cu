// Candidate token selection (LTD section 3.2, "Candidate Token Selection").
//
// One CTA per sequence.  Every node gets the key (cum desc, id asc) in
// shared memory (the root gets the maximum key, so it always ranks first);
// a bitonic sort of the keys (in registers and warp shuffles, one key per
// thread, up to 1024 nodes) puts the N verified nodes first (keys are
// unique, so the order is total).  A block-wide exclusive scan over the
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

// Optional phase timestamps for performance work (off in normal builds).
#ifdef LTD_TRACE
__device__ unsigned long long g_select_trace[64][8];
#define STRACE(slot)                                                            \
  do {                                                                          \
    if (threadIdx.x == 0 && blockIdx.x < 64) {                                  \
      unsigned long long t_;                                                    \
      asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t_));                   \
      g_select_trace[blockIdx.x][slot] = t_;                                    \
    }                                                                           \
  } while (0)
#else
#define STRACE(slot) \
  do {               \
  } while (0)
#endif

__global__ void __launch_bounds__(kNT) select_kernel(const SelectParams p) {
  extern __shared__ __align__(16) unsigned char smem[];
  const int W32 = (p.n_max + 31) / 32;
  const int P = p.sort_len;                                                   // pow2 >= max_nodes
  uint64_t* keys = reinterpret_cast<uint64_t*>(smem);                          // [P]
  int32_t* slot_of = reinterpret_cast<int32_t*>(keys + P);                    // [max_nodes]
  int32_t* par_s = slot_of + p.max_nodes;                                     // [max_nodes]
  uint32_t* words = reinterpret_cast<uint32_t*>(par_s + p.max_nodes);         // [n_max][W32]
  __shared__ int32_t warp_tot[kNT / kWarp];

  STRACE(0);
  grid_wait();
  trigger_dependents();
  STRACE(1);
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

  // keys padded to a power of two with 0 (below every real key)
  int Pn = 1;
  while (Pn < n) Pn <<= 1;
  for (int i = tid; i < n; i += kNT) {
    par_s[i] = p.parent[nb + i];
    slot_of[i] = 0;
  }
  for (int i = tid; i < p.n_max * W32; i += kNT) words[i] = 0u;
  const int lane = tid & 31, warp = tid >> 5;
  if (Pn <= kNT) {
    // one key per thread, bitonic sort descending: strides below the warp
    // width by shuffles, wider ones through shared memory
    uint64_t key = 0ull;
    if (tid < n) key = (tid == 0) ? ~0ull : make_key(p.cum[nb + tid], static_cast<uint32_t>(tid));
    __syncthreads();
    STRACE(2);
    // only warps holding keys compute; every thread meets the barriers
    const bool sorter = warp * kWarp < Pn;
    for (int k = 2; k <= Pn; k <<= 1) {
      for (int j = k >> 1; j > 0; j >>= 1) {
        uint64_t other = 0ull;
        if (j >= kWarp) {
          if (tid < Pn) keys[tid] = key;
          __syncthreads();
          if (tid < Pn) other = keys[tid ^ j];
          __syncthreads();
        } else if (sorter) {
          other = __shfl_xor_sync(0xFFFFFFFFu, key, j);
        }
        if (sorter) {
          // in a descending block the lower index of the pair keeps the larger
          const bool keep_max = ((tid & k) == 0) == ((tid & j) == 0);
          key = keep_max ? (key > other ? key : other) : (key < other ? key : other);
        }
      }
    }
    if (tid < N) slot_of[key_index(key)] = 1;
  } else {
    for (int i = tid; i < Pn; i += kNT)
      keys[i] = (i >= n) ? 0ull : (i == 0) ? ~0ull : make_key(p.cum[nb + i], static_cast<uint32_t>(i));
    __syncthreads();
    STRACE(2);
    for (int k = 2; k <= Pn; k <<= 1) {
      for (int j = k >> 1; j > 0; j >>= 1) {
        for (int i = tid; i < Pn; i += kNT) {
          const int ixj = i ^ j;
          if (ixj > i) {
            const uint64_t x = keys[i], y = keys[ixj];
            if (((i & k) == 0) ? (x < y) : (x > y)) {
              keys[i] = y;
              keys[ixj] = x;
            }
          }
        }
        __syncthreads();
      }
    }
    for (int r = tid; r < N; r += kNT) slot_of[key_index(keys[r])] = 1;
  }
  __syncthreads();
  STRACE(3);
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

  STRACE(4);
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
  STRACE(5);
}

}  // namespace

cudaError_t launch_select(const SelectParams& params, int32_t batch, cudaStream_t s) {
  SelectParams p = params;
  p.sort_len = 1;
  while (p.sort_len < p.max_nodes) p.sort_len <<= 1;
  const int W32 = (p.n_max + 31) / 32;
  const size_t smem = static_cast<size_t>(p.sort_len) * sizeof(uint64_t) +
                      static_cast<size_t>(p.max_nodes) * 2 * sizeof(int32_t) +
                      static_cast<size_t>(p.n_max) * W32 * sizeof(uint32_t);
  cudaError_t e = cudaFuncSetAttribute(select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  return launch(select_kernel, dim3(batch), dim3(kNT), smem, s, nullptr, 0, p);
}

#ifdef LTD_TRACE
extern "C" int ltd_select_trace_read(unsigned long long* host, int n) {
  return cudaMemcpyFromSymbol(host, g_select_trace, sizeof(unsigned long long) * n) == cudaSuccess ? 0
                                                                                                   : 1;
}
#endif

}  // namespace ltd
