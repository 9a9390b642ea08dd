// Observations of the two learned policies and the policies themselves
// (LTD section 3.1, "Reinforcement Learning Environment"; Appendix A.2,
// "Size Policy" and "Depth Policy").
//
// depth policy: after each expansion, the cumulative log-probabilities of the
// candidate tokens the current level produced (k^2 of them, k at level 1,
// padded to k^2), then the draft depth D and the sequence length L;
// size policy: the cumulative log-probabilities of every node of the tree
// (root included, padded to a fixed length), then D and L.
// The observation kernels (one CTA per sequence) gather from the tree arrays
// for a policy on the host; mlp_policy_kernel gathers them itself and runs
// the policy MLP on the device, writing the decision where the next launch
// of the cycle reads it.
#include <algorithm>

#include "ltd_common.cuh"
#include "ltd_internal.h"
#include "tc_util.cuh"

namespace ltd {

namespace {

// Split cluster barrier: every thread arrives (relaxed: no memory ordering)
// and later waits; between the two it may work on its own data.
__device__ __forceinline__ void cluster_arrive_relaxed() {
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() {
  asm volatile("barrier.cluster.wait.aligned;" ::: "memory");
}

constexpr int kPolicyNT = 256;

__global__ void __launch_bounds__(kPolicyNT) depth_obs_kernel(const ltd_tree t, const int32_t* ctx,
                                                              float* out) {
  grid_wait();
  trigger_dependents();
  const int b = blockIdx.x;
  const int k = t.k, kk = k * k;
  const int lvl = t.n_levels[b];
  const int64_t nb = static_cast<int64_t>(b) * t.max_nodes;
  // the level's candidates: ids 1..k at level 1, k^2 ids from 1 + k + (l-2) k^2 after
  const int first = (lvl <= 1) ? 1 : 1 + k + (lvl - 2) * kk;
  const int count = (lvl < 1) ? 0 : ((lvl == 1) ? k : kk);
  float* o = out + static_cast<int64_t>(b) * (kk + 2);
  for (int i = threadIdx.x; i < kk; i += kPolicyNT)
    o[i] = (i < count) ? __ldcg(&t.cum_logprob[nb + first + i]) : kPolicyPad;
  if (threadIdx.x == 0) {
    o[kk] = static_cast<float>(lvl);
    o[kk + 1] = static_cast<float>(ctx[b]);
  }
}

__global__ void __launch_bounds__(kPolicyNT) size_obs_kernel(const ltd_tree t, const int32_t* ctx,
                                                             int32_t v_pad, float* out) {
  grid_wait();
  trigger_dependents();
  const int b = blockIdx.x;
  const int n = t.n_nodes[b];
  const int64_t nb = static_cast<int64_t>(b) * t.max_nodes;
  float* o = out + static_cast<int64_t>(b) * (v_pad + 2);
  for (int i = threadIdx.x; i < v_pad; i += kPolicyNT)
    o[i] = (i < n) ? __ldcg(&t.cum_logprob[nb + i]) : kPolicyPad;
  if (threadIdx.x == 0) {
    o[v_pad] = static_cast<float>(t.n_levels[b]);
    o[v_pad + 1] = static_cast<float>(ctx[b]);
  }
}

// ------------------------------------------------ policies on the device
// One thread-block cluster of kMlpC CTAs (on the SMs of one GPC) evaluates
// the MLP for groups of up to kMlpG sequences at a time, so every weight is
// read once per group.  Each CTA owns a slice of every layer's output units;
// a thread owns a quad of four consecutive units and every P-th input row,
// the P partial sums of a unit being added in a fixed order.  A packed
// network (ltd_mlp_pack: every CTA's column slice of W stored contiguously)
// streams the slice through a ring of shared-memory stages, one bulk copy
// of up to kMlpStageBytes per stage, issued up to kMlpStages stages ahead
// (also across layers), so the whole slice is in flight at once; a
// row-major network is read with plain loads.  Each layer's outputs are
// pushed into every CTA's next activation buffer through distributed shared
// memory, and one cluster barrier per layer publishes them.
#ifdef LTD_TRACE
__device__ unsigned long long g_mlp_trace[16][16];
__device__ unsigned long long g_mlp_chunk_trace[16][64];  // per chunk: issued, landed
#define CTRACE(slot)                                                            \
  do {                                                                          \
    unsigned long long t_;                                                      \
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t_));                     \
    if ((slot) < 64) g_mlp_chunk_trace[blockIdx.x & 15][(slot) & 63] = t_;      \
  } while (0)
#define MTRACE(slot)                                             \
  do {                                                           \
    unsigned long long t_;                                       \
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t_));      \
    if (threadIdx.x == 0) g_mlp_trace[blockIdx.x & 15][slot] = t_; \
  } while (0)
#else
#define MTRACE(slot) \
  do {               \
  } while (0)
#define CTRACE(slot) \
  do {               \
  } while (0)
#endif

constexpr int kMlpC = 16;  // CTAs per cluster (non-portable size)
constexpr int kMlpNT = 256;
constexpr int kMlpG = 8;
constexpr int kMlpStages = 4;
constexpr int kMlpStageBytes = 32 * 1024;
constexpr int kMlpBiasMax = LTD_MLP_MAX_WIDTH / kMlpC + 4;  // units of a CTA in one layer

struct MlpLayerPlan {
  int32_t U;     // units per CTA (the stage row stride, in floats)
  int32_t bulk;  // 1: streamed through the ring; 0: direct loads
  int32_t R;     // rows per chunk (bulk layers)
};

struct MlpArgs {
  ltd_tree t;
  const int32_t* ctx;
  ltd_mlp net;
  MlpLayerPlan plan[LTD_MLP_MAX_LAYERS];
  int32_t size_policy;  // 0: depth policy, 1: size policy
  int32_t v_pad;        // size policy: padded score count
  const int32_t* active_in;
  int32_t* active_out;
  int32_t n_cap;
  int32_t* n_verify;
  float* logits;
  uint32_t* err;
  int32_t G;      // sequences per group
  int32_t width;  // row stride of an activation buffer (largest width)
};

__device__ __forceinline__ void gather_obs(const MlpArgs& a, int b, float* x) {
  const ltd_tree& t = a.t;
  const int64_t nb = static_cast<int64_t>(b) * t.max_nodes;
  const int lvl = t.n_levels[b];
  if (a.size_policy) {
    const int n = t.n_nodes[b];
    for (int i = threadIdx.x; i < a.v_pad; i += kMlpNT)
      x[i] = (i < n) ? __ldcg(&t.cum_logprob[nb + i]) : kPolicyPad;
    if (threadIdx.x == 0) {
      x[a.v_pad] = static_cast<float>(lvl);
      x[a.v_pad + 1] = static_cast<float>(a.ctx[b]);
    }
  } else {
    const int k = t.k, kk = k * k;
    const int first = (lvl <= 1) ? 1 : 1 + k + (lvl - 2) * kk;
    const int count = (lvl < 1) ? 0 : ((lvl == 1) ? k : kk);
    for (int i = threadIdx.x; i < kk; i += kMlpNT)
      x[i] = (i < count) ? __ldcg(&t.cum_logprob[nb + first + i]) : kPolicyPad;
    if (threadIdx.x == 0) {
      x[kk] = static_cast<float>(lvl);
      x[kk + 1] = static_cast<float>(a.ctx[b]);
    }
  }
}

// Chunks a CTA streams for layer l: ceil(n_in / R) when the layer is bulk
// and this CTA owns units of it, else none.
__device__ __forceinline__ int layer_chunks(const MlpArgs& a, int l, int rank) {
  const MlpLayerPlan& pl = a.plan[l];
  if (!pl.bulk) return 0;
  const int n_out = a.net.dims[l + 1];
  if (rank * pl.U >= n_out) return 0;
  return (a.net.dims[l] + pl.R - 1) / pl.R;
}

// Thread 0 issues chunk `c` (flat index over groups and layers) into its stage.
__device__ __forceinline__ void issue_chunk(const MlpArgs& a, int c, int per_group, int rank,
                                            uint32_t ring, uint32_t bars) {
  int j = c % per_group, l = 0;
  for (; l < a.net.n_layers; ++l) {
    const int n = layer_chunks(a, l, rank);
    if (j < n) break;
    j -= n;
  }
  const MlpLayerPlan& pl = a.plan[l];
  const int n_in = a.net.dims[l];
  const int r0 = j * pl.R;
  const int rows = min(pl.R, n_in - r0);
  const int s = c % kMlpStages;
  const uint32_t bar = bars + 8u * s;
  const uint32_t bytes = static_cast<uint32_t>(rows * pl.U) * 4u;
  CTRACE(2 * c);
  tc::mbar_expect_tx(bar, bytes);
  tc::bulk_g2s(ring + static_cast<uint32_t>(s) * kMlpStageBytes,
               a.net.w[l] + (static_cast<int64_t>(rank) * n_in + r0) * pl.U, bytes, bar);
}

// G: sequences per group (the accumulators of a thread); a group with fewer
// sequences computes the missing ones on unused buffer rows and drops them.
template <int G>
__global__ void __launch_bounds__(kMlpNT, 1) mlp_policy_kernel(const MlpArgs a) {
  extern __shared__ __align__(128) unsigned char mlp_smem[];
  const uint32_t ring = tc::smem_u32(mlp_smem);
  float* const act0 = reinterpret_cast<float*>(mlp_smem + kMlpStages * kMlpStageBytes);
  const int act_stride = G * a.width;        // two [G][width] activation buffers
  float* const red = act0 + 2 * act_stride;  // [kMlpNT][G][4] partial sums
  float* const bias_s = red + kMlpNT * G * 4;  // [layer][kMlpBiasMax] this CTA's biases
  uint64_t* const bar_p = reinterpret_cast<uint64_t*>(bias_s + LTD_MLP_MAX_LAYERS * kMlpBiasMax);
  const uint32_t bars = tc::smem_u32(bar_p);
  const int tid = threadIdx.x;
  const int rank = static_cast<int>(tc::cluster_rank());
  const int B = a.t.batch;
  const int L = a.net.n_layers;
  const int n_groups = (B + G - 1) / G;
  int per_group = 0;
  for (int l = 0; l < L; ++l) per_group += layer_chunks(a, l, rank);
  const int total = per_group * n_groups;
  MTRACE(0);
  if (tid == 0) {
    for (int s = 0; s < kMlpStages; ++s) tc::mbar_init(bars + 8u * s, 1);
    tc::mbar_init_fence();
  }
  __syncthreads();
  // the weights do not depend on earlier kernels: start streaming them
  int issued = min(kMlpStages, total);
  if ((tid & 31) == 0 && (tid >> 5) < issued) issue_chunk(a, tid >> 5, per_group, rank, ring, bars);
  // this CTA's biases (a few hundred floats) to shared memory, off the
  // critical path of the unit sums
  for (int l = 0; l < L; ++l) {
    const int U = a.plan[l].U, u0 = rank * U;
    const int u_cnt = max(0, min(U, a.net.dims[l + 1] - u0));
    for (int u = tid; u < u_cnt; u += kMlpNT) bias_s[l * kMlpBiasMax + u] = __ldcg(a.net.b[l] + u0 + u);
  }
  // peers must have started before their shared memory is written
  cluster_arrive_relaxed();
  bool peers_known = false;
  MTRACE(1);
  grid_wait();
  trigger_dependents();
  MTRACE(2);
  int consumed = 0;
  bool timed_out = false;
  for (int b0 = 0; b0 < B; b0 += G) {
    const int gn = min(G, B - b0);
    for (int g = 0; g < gn; ++g) gather_obs(a, b0 + g, act0 + g * a.width);
    __syncthreads();
    MTRACE(3);
    int cur = 0;
    for (int l = 0; l < L; ++l) {
      const MlpLayerPlan pl = a.plan[l];
      const int n_in = a.net.dims[l], n_out = a.net.dims[l + 1];
      const int U = pl.U;
      const int u0 = rank * U;
      const int u_cnt = max(0, min(U, n_out - u0));
      // a thread owns a quad of 4 consecutive units and every P-th input row
      const int Q = (U + 3) >> 2;
      int Qp = 1;
      while (Qp < Q) Qp <<= 1;
      const int P = kMlpNT / Qp;
      const int q = tid % Qp, p = tid / Qp;
      const bool valid = 4 * q < u_cnt;
      const float* x = act0 + cur * act_stride;
      float acc[G][4];
#pragma unroll
      for (int g = 0; g < G; ++g)
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[g][c] = 0.f;
      if (pl.bulk) {
        const int nch = layer_chunks(a, l, rank);
        for (int j = 0; j < nch; ++j, ++consumed) {
          const int s = consumed % kMlpStages;
          if (!timed_out && !tc::mbar_wait(bars + 8u * s, (consumed / kMlpStages) & 1)) {
            timed_out = true;
            if (tid == 0) flag_error(a.err, LTD_DEVERR_TIMEOUT);
          }
          if (tid == 0) CTRACE(2 * consumed + 1);
          const float4* st = reinterpret_cast<const float4*>(mlp_smem + s * kMlpStageBytes);
          const int r0 = j * pl.R;
          const int rows = min(pl.R, n_in - r0);
          if (valid) {
            const int q4 = U >> 2;
#pragma unroll 4
            for (int r = p; r < rows; r += P) {
              const float4 w = st[r * q4 + q];
#pragma unroll
              for (int g = 0; g < G; ++g) {
                const float xv = x[g * a.width + r0 + r];
                acc[g][0] = fmaf(xv, w.x, acc[g][0]);
                acc[g][1] = fmaf(xv, w.y, acc[g][1]);
                acc[g][2] = fmaf(xv, w.z, acc[g][2]);
                acc[g][3] = fmaf(xv, w.w, acc[g][3]);
              }
            }
          }
          __syncthreads();  // stage s is free again
          if (issued < total && tid == 0) issue_chunk(a, issued, per_group, rank, ring, bars);
          ++issued;
        }
      } else if (valid) {
        const float* wq = a.net.w[l] + u0 + 4 * q;
        const int nc = min(4, u_cnt - 4 * q);
        for (int i = p; i < n_in; i += P) {
          float w[4];
#pragma unroll
          for (int c = 0; c < 4; ++c) w[c] = (c < nc) ? __ldcg(wq + static_cast<int64_t>(i) * n_out + c) : 0.f;
#pragma unroll
          for (int g = 0; g < G; ++g) {
            const float xv = x[g * a.width + i];
#pragma unroll
            for (int c = 0; c < 4; ++c) acc[g][c] = fmaf(xv, w[c], acc[g][c]);
          }
        }
      }
#pragma unroll
      for (int g = 0; g < G; ++g)
        *reinterpret_cast<float4*>(red + (tid * G + g) * 4) =
            make_float4(acc[g][0], acc[g][1], acc[g][2], acc[g][3]);
      __syncthreads();
      MTRACE(4 + 2 * l);
      // unit sums in a fixed order, then the push to every CTA
      const bool hidden = l + 1 < L;
      float* nxt = act0 + (cur ^ 1) * act_stride;
      const int n_outs = u_cnt * gn;
      const float* bl = bias_s + l * kMlpBiasMax;
      if (!peers_known) {
        cluster_wait();
        peers_known = true;
      }
      // a unit sum adds P partials: one thread per unit when there are many
      // units, a warp per unit when there are few units with many partials
      // (estimated cycles of each)
      const int serial_cost = ((n_outs + kMlpNT - 1) / kMlpNT) * P;
      const int warp_cost = ((n_outs + kMlpNT / 32 - 1) / (kMlpNT / 32)) * ((P + 31) / 32 + 7);
      if (warp_cost < serial_cost) {
        // many partials per unit: a warp per unit, lanes over the partials
        const int lane = tid & 31;
        for (int o = tid >> 5; o < n_outs; o += kMlpNT / 32) {
          const int u = o % u_cnt, g = o / u_cnt;
          const int uq = u >> 2, uc = u & 3;
          float part = 0.f;
          for (int pp = lane; pp < P; pp += 32) part += red[((pp * Qp + uq) * G + g) * 4 + uc];
#pragma unroll
          for (int off = 16; off > 0; off >>= 1) part += __shfl_xor_sync(0xffffffffu, part, off);
          float sum = bl[u] + part;
          if (hidden) sum = fmaxf(sum, 0.f);
          if (lane < kMlpC)
            tc::st_cluster_f1(tc::mapa(tc::smem_u32(nxt + g * a.width + u0 + u), lane), sum);
        }
      } else {
        for (int idx = tid; idx < n_outs; idx += kMlpNT) {
          const int u = idx % u_cnt, g = idx / u_cnt;
          const int uq = u >> 2, uc = u & 3;
          float sum = bl[u];
          for (int pp = 0; pp < P; ++pp) sum += red[((pp * Qp + uq) * G + g) * 4 + uc];
          if (hidden) sum = fmaxf(sum, 0.f);
          const uint32_t local = tc::smem_u32(nxt + g * a.width + u0 + u);
          for (uint32_t r = 0; r < static_cast<uint32_t>(kMlpC); ++r)
            tc::st_cluster_f1(tc::mapa(local, r), sum);
        }
      }
      tc::cluster_sync();
      MTRACE(5 + 2 * l);
      cur ^= 1;
    }
    // every CTA now holds the logits; rank 0 decides
    if (rank == 0 && tid < gn) {
      const int b = b0 + tid;
      const int n_act = a.net.dims[L];
      const float* z = act0 + cur * act_stride + tid * a.width;
      int best = 0;
      for (int j = 1; j < n_act; ++j)
        if (z[j] > z[best]) best = j;  // ties keep the lower action
      if (a.logits != nullptr)
        for (int j = 0; j < n_act; ++j) a.logits[static_cast<int64_t>(b) * n_act + j] = z[j];
      if (a.size_policy) {
        const int v = 20 + 20 * best;
        a.n_verify[b] = min(min(1 + v, a.n_cap), a.t.n_nodes[b]);
      } else {
        const bool was = a.active_in == nullptr || a.active_in[b] != 0;
        a.active_out[b] = (was && best == 1 && a.t.n_levels[b] < a.t.max_depth) ? 1 : 0;
      }
    }
    MTRACE(12);
    // the group's buffers are rewritten by the next group (after the last
    // group no CTA touches another's shared memory any more)
    if (b0 + G < B) tc::cluster_sync();
  }
  MTRACE(13);
}

// packed[r][i][u] = W[i][r U + u] for the columns that exist, else 0.
__global__ void __launch_bounds__(256) mlp_pack_kernel(const float* __restrict__ w, int32_t n_in,
                                                       int32_t n_out, int32_t U, float* out) {
  grid_wait();
  trigger_dependents();
  const int64_t total = static_cast<int64_t>(kMlpC) * n_in * U;
  for (int64_t idx = blockIdx.x * 256ll + threadIdx.x; idx < total; idx += gridDim.x * 256ll) {
    const int64_t slice = static_cast<int64_t>(n_in) * U;
    const int r = static_cast<int>(idx / slice);
    const int64_t rem = idx - r * slice;
    const int i = static_cast<int>(rem / U), u = static_cast<int>(rem % U);
    const int col = r * U + u;
    out[idx] = (col < n_out) ? w[static_cast<int64_t>(i) * n_out + col] : 0.f;
  }
}

}  // namespace

int mlp_packed_units(int n_out) { return ((n_out + kMlpC - 1) / kMlpC + 3) & ~3; }

size_t mlp_packed_floats(const ltd_mlp* net, size_t offsets[LTD_MLP_MAX_LAYERS]) {
  size_t total = 0;
  for (int l = 0; l < net->n_layers; ++l) {
    offsets[l] = total;
    const size_t n = static_cast<size_t>(kMlpC) * net->dims[l] * mlp_packed_units(net->dims[l + 1]);
    total += (n + 63) & ~static_cast<size_t>(63);  // every matrix 256-byte aligned
  }
  return total;
}

cudaError_t launch_mlp_pack(const ltd_mlp* net, float* base, ltd_mlp* packed, cudaStream_t s) {
  size_t off[LTD_MLP_MAX_LAYERS];
  mlp_packed_floats(net, off);
  *packed = *net;
  packed->layout = LTD_MLP_PACKED;
  for (int l = 0; l < net->n_layers; ++l) {
    const int U = mlp_packed_units(net->dims[l + 1]);
    float* out = base + off[l];
    packed->w[l] = out;
    const int64_t total = static_cast<int64_t>(kMlpC) * net->dims[l] * U;
    const int blocks = static_cast<int>(std::min<int64_t>((total + 255) / 256, 1024));
    cudaError_t e = launch(mlp_pack_kernel, dim3(blocks), dim3(256), 0, s, nullptr, 0, net->w[l],
                           net->dims[l], net->dims[l + 1], U, out);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

cudaError_t launch_mlp_policy(const ltd_tree* t, const int32_t* ctx, const ltd_mlp* net,
                              int32_t size_policy, int32_t v_pad, const int32_t* active_in,
                              int32_t* active_out, int32_t n_cap, int32_t* n_verify,
                              float* logits, cudaStream_t s) {
  MlpArgs a = {};
  a.t = *t;
  a.ctx = ctx;
  a.net = *net;
  a.size_policy = size_policy;
  a.v_pad = v_pad;
  a.active_in = active_in;
  a.active_out = active_out;
  a.n_cap = n_cap;
  a.n_verify = n_verify;
  a.logits = logits;
  a.err = device_error_word();
  if (a.err == nullptr) return cudaErrorUnknown;
  int width = 0;
  for (int l = 0; l <= net->n_layers; ++l) width = std::max(width, static_cast<int>(net->dims[l]));
  width = (width + 3) & ~3;  // keep every buffer row 16-byte aligned
  a.width = width;
  const bool packed = net->layout == LTD_MLP_PACKED;
  for (int l = 0; l < net->n_layers; ++l) {
    const int n_out = net->dims[l + 1];
    MlpLayerPlan& pl = a.plan[l];
    pl.U = packed ? mlp_packed_units(n_out) : (n_out + kMlpC - 1) / kMlpC;
    pl.bulk = packed ? 1 : 0;
    pl.R = packed ? kMlpStageBytes / (pl.U * 4) : 0;
  }
  // as many sequences per group as fit in shared memory (a power of two)
  constexpr size_t kBudget = 227 * 1024;
  const size_t fixed = static_cast<size_t>(kMlpStages) * kMlpStageBytes +
                       LTD_MLP_MAX_LAYERS * kMlpBiasMax * sizeof(float) + kMlpStages * 8;
  const size_t per_seq = (2 * static_cast<size_t>(width) + 4 * kMlpNT) * sizeof(float);
  if (kBudget < fixed + per_seq) return cudaErrorInvalidValue;
  const size_t fit = std::min<size_t>(kMlpG, (kBudget - fixed) / per_seq);
  int G = 1;
  while (G < t->batch && static_cast<size_t>(2 * G) <= fit) G <<= 1;
  a.G = G;
  const size_t smem = fixed + per_seq * G;
  void (*kern)(MlpArgs) = G == 1   ? mlp_policy_kernel<1>
                          : G == 2 ? mlp_policy_kernel<2>
                          : G == 4 ? mlp_policy_kernel<4>
                                   : mlp_policy_kernel<8>;
  cudaError_t e =
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e != cudaSuccess) return e;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = kMlpC;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  return launch(kern, dim3(kMlpC), dim3(kMlpNT), smem, s, attr, 1, a);
}

#ifdef LTD_TRACE
extern "C" int ltd_mlp_trace_read(unsigned long long* host) {
  return cudaMemcpyFromSymbol(host, g_mlp_trace, sizeof(g_mlp_trace)) == cudaSuccess ? 0 : 1;
}
extern "C" int ltd_mlp_chunk_trace_read(unsigned long long* host) {
  return cudaMemcpyFromSymbol(host, g_mlp_chunk_trace, sizeof(g_mlp_chunk_trace)) == cudaSuccess
             ? 0
             : 1;
}
#endif

cudaError_t launch_depth_obs(const ltd_tree* t, const int32_t* ctx, float* out, cudaStream_t s) {
  return launch(depth_obs_kernel, dim3(t->batch), dim3(kPolicyNT), 0, s, nullptr, 0, *t, ctx, out);
}

cudaError_t launch_size_obs(const ltd_tree* t, const int32_t* ctx, int32_t v_pad, float* out,
                            cudaStream_t s) {
  return launch(size_obs_kernel, dim3(t->batch), dim3(kPolicyNT), 0, s, nullptr, 0, *t, ctx, v_pad,
                out);
}

}  // namespace ltd
