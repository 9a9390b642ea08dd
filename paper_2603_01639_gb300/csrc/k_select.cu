// Candidate token selection (LTD section 3.2, "Candidate Token Selection").
//
// One CTA per sequence.  Every node gets the key (cum desc, id asc); the
// root gets the largest key, so it always ranks first.  The N largest keys
// are found by a radix select over the 64-bit keys, eight bits per pass
// from the top: a shared-memory histogram of the next digit among the keys
// that match the prefix so far, one warp's scan of it from the top bin, and
// the bin where the count reaches N becomes the prefix; the select stops at
// the first pass whose bin holds exactly the keys still wanted (keys are
// unique, so it stops by the last digit), and a key is verified iff its
// bits above that digit are at least the prefix.  Typically three passes.
// Slots are the verified ids in ascending order (a block scan of the
// flags).  The thread that owns a verified node walks its parent chain (at
// most max_depth steps) and builds the node's mask row in registers, one
// bit per ancestor, then stores it.  Because a child's cum never exceeds its
// parent's and parents have smaller ids, the verified set is
// ancestor-closed; a violation is flagged, not trapped.
#include "ltd_common.cuh"
#include "ltd_internal.h"

namespace ltd {

namespace {

constexpr int kNT = 1024;
constexpr int kNW = kNT / kWarp;
constexpr int kMaxPer = LTD_MAX_TREE_NODES / kNT;  // nodes per thread
constexpr int kMaxWords = LTD_MAX_N / 32;          // mask words per row
static_assert(LTD_MAX_TREE_NODES % kNT == 0, "whole nodes per thread");

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

struct RadixState {
  uint64_t prefix;  // the selected digits so far
  int shift;        // bit position of the current digit
  int want;         // keys still to select among those matching the prefix
  int done;
};

__global__ void __launch_bounds__(kNT) select_kernel(const SelectParams p) {
  extern __shared__ __align__(16) unsigned char smem[];
  int32_t* slot_of = reinterpret_cast<int32_t*>(smem);  // [max_nodes]
  int32_t* par_s = slot_of + p.max_nodes;               // [max_nodes]
  __shared__ uint32_t hist[2][256];
  __shared__ int warp_tot[kNW];
  __shared__ RadixState st;

  STRACE(0);
  const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (int i = tid; i < 512; i += kNT) (&hist[0][0])[i] = 0u;
  grid_wait();
  trigger_dependents();
  STRACE(1);
  const int64_t nb = static_cast<int64_t>(b) * p.max_nodes;
  const int W32 = (p.n_max + 31) / 32;
  int32_t* ids_out = p.node_ids + static_cast<int64_t>(b) * p.n_max;
  int32_t* pos_out = p.pos + static_cast<int64_t>(b) * p.n_max;
  uint32_t* mask_out = p.mask + static_cast<int64_t>(b) * p.n_max * W32;

  // every node slot's data is loaded before the node count is known
  const int per = (p.max_nodes + kNT - 1) / kNT;
  float cumv[kMaxPer];
  int parv[kMaxPer], depv[kMaxPer];
#pragma unroll
  for (int q = 0; q < kMaxPer; ++q) {
    const int i = tid + q * kNT;
    cumv[q] = 0.f;
    parv[q] = -1;
    depv[q] = 0;
    if (q < per && i < p.max_nodes) {
      cumv[q] = __ldcg(p.cum + nb + i);
      parv[q] = __ldcg(p.parent + nb + i);
      depv[q] = __ldcg(p.depth + nb + i);
    }
  }
  const int n = __ldcg(p.n_nodes + b);
  const int N = __ldcg(p.n_verify + b);
  const int ctx = __ldcg(p.ctx + b);

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
  // slots past N (known already)
  for (int i = N + tid; i < p.n_max; i += kNT) {
    ids_out[i] = -1;
    pos_out[i] = -1;
  }
  for (int i = N * W32 + tid; i < p.n_max * W32; i += kNT) mask_out[i] = 0u;

  uint64_t key[kMaxPer];
#pragma unroll
  for (int q = 0; q < kMaxPer; ++q) {
    const int i = tid + q * kNT;
    key[q] = (q < per && i < n) ? ((i == 0) ? ~0ull : make_key(cumv[q], static_cast<uint32_t>(i))) : 0ull;
    if (q < per && i < n) par_s[i] = parv[q];
  }
  if (tid == 0) {
    st.prefix = 0ull;
    st.shift = 56;
    st.want = N;
    st.done = 0;
  }
  __syncthreads();
  STRACE(2);

  // ---- radix select of the N largest keys (key 0 = no node)
#pragma unroll 1
  for (int pass = 0; pass < 8; ++pass) {
    const int buf = pass & 1;
    const int shift = st.shift;
    const uint64_t prefix = st.prefix;
#pragma unroll
    for (int q = 0; q < kMaxPer; ++q) {
      if (q >= per) break;
      const bool match = key[q] != 0ull && (pass == 0 || (key[q] >> (shift + 8)) == prefix);
      const uint32_t dig = match ? static_cast<uint32_t>(key[q] >> shift) & 0xFFu : 0x100u;
      const uint32_t peers = __match_any_sync(0xFFFFFFFFu, dig);
      if (dig < 256u && lane == __ffs(peers) - 1) atomicAdd(&hist[buf][dig], __popc(peers));
    }
    __syncthreads();
    if (warp == 0) {
      // lane l covers bins 255 - 8l - j, j = 0..7 (from the top)
      uint32_t c[8];
      uint32_t s = 0u;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        c[j] = hist[buf][255 - 8 * lane - j];
        s += c[j];
      }
      uint32_t incl = s;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
        if (lane >= o) incl += y;
      }
      const uint32_t want = static_cast<uint32_t>(st.want);
      const uint32_t before = incl - s;
      // exactly one lane's range crosses `want`
      if (before < want && incl >= want) {
        // the first of the lane's bins where the count reaches want (the
        // lane's total does)
        uint32_t above = before, cj = 0u;
        int j = 0;
        bool found = false;
#pragma unroll
        for (int jj = 0; jj < 8; ++jj) {
          if (!found) {
            if (above + c[jj] >= want) {
              j = jj;
              cj = c[jj];
              found = true;
            } else {
              above += c[jj];
            }
          }
        }
        const uint32_t bin = 255u - 8u * lane - j;
        const uint32_t rest = want - above;
        st.prefix = (prefix << 8) | bin;
        st.want = static_cast<int>(rest);
        if (cj == rest || shift == 0) {
          st.done = 1;
        } else {
          st.shift = shift - 8;
        }
      }
      // the other buffer is clean for the next pass
#pragma unroll
      for (int j = 0; j < 8; ++j) hist[buf ^ 1][8 * lane + j] = 0u;
    }
    __syncthreads();
    if (st.done) break;
  }
  STRACE(3);
  const int fshift = st.shift;
  const uint64_t thresh = st.prefix;

  // ---- slots: verified ids in ascending order (id = tid + q * kNT)
  int slot_base = 0;
  int my_slot[kMaxPer];
#pragma unroll
  for (int q = 0; q < kMaxPer; ++q) {
    my_slot[q] = -1;
    if (q >= per) break;
    const bool sel = key[q] != 0ull && (key[q] >> fshift) >= thresh;
    const uint32_t bal = __ballot_sync(0xFFFFFFFFu, sel);
    if (lane == 0) warp_tot[warp] = __popc(bal);
    __syncthreads();
    const int t = warp_tot[lane];
    int incl = t;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
      if (lane >= o) incl += y;
    }
    const int warp_before = __shfl_sync(0xFFFFFFFFu, incl - t, warp);
    const int total = __shfl_sync(0xFFFFFFFFu, incl, 31);
    const int i = tid + q * kNT;
    if (sel) {
      const int s = slot_base + warp_before + __popc(bal & ((1u << lane) - 1u));
      my_slot[q] = s;
      ids_out[s] = i;
      pos_out[s] = ctx + depv[q];
    }
    if (q < per && i < n) slot_of[i] = my_slot[q];
    slot_base += total;
    __syncthreads();  // warp_tot is reused by the next q
  }
  STRACE(4);

  // ---- mask rows: the owner of a verified node walks its parent chain
#pragma unroll
  for (int q = 0; q < kMaxPer; ++q) {
    if (q >= per) break;
    const int si = my_slot[q];
    if (si < 0) continue;
    uint32_t row[kMaxWords];
#pragma unroll
    for (int w = 0; w < kMaxWords; ++w) row[w] = 0u;
    int a = tid + q * kNT;
    int guard = 0;
    while (a >= 0 && guard <= LTD_MAX_DEPTH + 1) {
      const int sa = (a < n) ? slot_of[a] : -1;
      if (sa < 0) {
        flag_error(p.err, LTD_DEVERR_TREE);
        break;
      }
#pragma unroll
      for (int w = 0; w < kMaxWords; ++w) row[w] |= ((sa >> 5) == w) ? (1u << (sa & 31)) : 0u;
      a = par_s[a];
      ++guard;
    }
    uint32_t* dst = mask_out + static_cast<int64_t>(si) * W32;
#pragma unroll
    for (int w = 0; w < kMaxWords; ++w)
      if (w < W32) dst[w] = row[w];
  }
  STRACE(5);
}

}  // namespace

cudaError_t launch_select(const SelectParams& params, int32_t batch, cudaStream_t s) {
  SelectParams p = params;
  const size_t smem = static_cast<size_t>(p.max_nodes) * 2 * sizeof(int32_t);
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
