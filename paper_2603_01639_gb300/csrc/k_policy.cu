// Observations of the two learned policies (LTD section 3.1, "Reinforcement
// Learning Environment"; Appendix A, "Observation Space").
//
// depth policy: after each expansion, the cumulative log-probabilities of the
// candidate tokens the current level produced (k^2 of them, k at level 1,
// padded to k^2), then the draft depth D and the sequence length L;
// size policy: the cumulative log-probabilities of every node of the tree
// (root included, padded to a fixed length), then D and L.
// One CTA per sequence gathers from the tree arrays; the policies themselves
// run on the host.
#include "ltd_common.cuh"
#include "ltd_internal.h"

namespace ltd {

namespace {

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

}  // namespace

cudaError_t launch_depth_obs(const ltd_tree* t, const int32_t* ctx, float* out, cudaStream_t s) {
  return launch(depth_obs_kernel, dim3(t->batch), dim3(kPolicyNT), 0, s, nullptr, 0, *t, ctx, out);
}

cudaError_t launch_size_obs(const ltd_tree* t, const int32_t* ctx, int32_t v_pad, float* out,
                            cudaStream_t s) {
  return launch(size_obs_kernel, dim3(t->batch), dim3(kPolicyNT), 0, s, nullptr, 0, *t, ctx, v_pad,
                out);
}

}  // namespace ltd
