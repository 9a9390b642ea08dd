// C ABI glue: argument validation, memory carving and kernel launches for the
// entry points declared in include/ltd.h.  Nothing here allocates device
// memory; the per-device error word is a file-scope __device__ variable.
#include <cuda_runtime.h>

#include <cstdlib>
#include <mutex>

#include <nvtx3/nvToolsExt.h>

#include "ltd.h"
#include "ltd_internal.h"

namespace ltd {

__device__ uint32_t g_error_word;

uint32_t* device_error_word() {
  static std::mutex mu;
  static uint32_t* ptrs[128] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 128) return nullptr;
  std::lock_guard<std::mutex> lock(mu);
  if (ptrs[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_error_word) != cudaSuccess) return nullptr;
    ptrs[dev] = static_cast<uint32_t*>(p);
  }
  return ptrs[dev];
}

bool pdl_enabled() {
  static const bool on = [] {
    const char* v = std::getenv("LTD_NO_PDL");
    return !(v != nullptr && v[0] == '1');
  }();
  return on;
}

namespace {

size_t align256(size_t x) { return (x + 255) / 256 * 256; }

size_t dtype_size(ltd_dtype d) { return d == LTD_BF16 ? 2 : 4; }

bool dtype_ok(ltd_dtype d) { return d == LTD_F32 || d == LTD_BF16; }

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int64_t tree_nodes(int32_t max_depth, int32_t k) {
  return 1 + static_cast<int64_t>(k) + static_cast<int64_t>(max_depth - 1) * k * k;
}

bool tree_dims_ok(int32_t batch, int32_t max_depth, int32_t k, int64_t max_vocab) {
  return batch >= 1 && max_depth >= 1 && max_depth <= LTD_MAX_DEPTH && k >= 1 &&
         k <= LTD_MAX_K && max_vocab >= k && max_vocab <= 0x7FFFFFFF &&
         tree_nodes(max_depth, k) <= LTD_MAX_TREE_NODES;
}

bool tree_ok(const ltd_tree* t) {
  return t != nullptr && tree_dims_ok(t->batch, t->max_depth, t->k, t->max_vocab) &&
         t->max_nodes == tree_nodes(t->max_depth, t->k) && t->token && t->parent && t->depth &&
         t->cum_logprob && t->xrow && t->xlse && t->frontier && t->n_nodes && t->n_levels &&
         t->scratch;
}

ltd_status from_cuda(cudaError_t e) { return e == cudaSuccess ? LTD_OK : LTD_ERR_CUDA; }

}  // namespace

bool tree_valid(const ltd_tree* t) { return tree_ok(t); }

}  // namespace ltd

using namespace ltd;

namespace {
// An NVTX range over one API call (named after it), so a profiler can
// attribute the kernels a call launches; without a tool attached the calls
// are no-ops.
struct ApiRange {
  explicit ApiRange(const char* name) { nvtxRangePushA(name); }
  ~ApiRange() { nvtxRangePop(); }
  ApiRange(const ApiRange&) = delete;
  ApiRange& operator=(const ApiRange&) = delete;
};
}  // namespace

extern "C" {

int32_t ltd_version(void) { return 100; }

const char* ltd_status_string(ltd_status s) {
  switch (s) {
    case LTD_OK: return "LTD_OK";
    case LTD_ERR_INVALID_ARG: return "LTD_ERR_INVALID_ARG";
    case LTD_ERR_SHAPE: return "LTD_ERR_SHAPE";
    case LTD_ERR_UNSUPPORTED: return "LTD_ERR_UNSUPPORTED";
    case LTD_ERR_CUDA: return "LTD_ERR_CUDA";
    case LTD_ERR_DEVICE: return "LTD_ERR_DEVICE";
    case LTD_ERR_TIMEOUT: return "LTD_ERR_TIMEOUT";
  }
  return "LTD_ERR_UNKNOWN";
}

size_t ltd_tree_bytes(int32_t batch, int32_t max_depth, int32_t k, int64_t max_vocab) {
  if (!tree_dims_ok(batch, max_depth, k, max_vocab)) return 0;
  const size_t nodes = static_cast<size_t>(batch) * tree_nodes(max_depth, k);
  return 6 * align256(nodes * 4) + align256(static_cast<size_t>(batch) * k * 4) +
         2 * align256(static_cast<size_t>(batch) * 4) + expand_scratch_bytes(batch, k, max_vocab);
}

ltd_status ltd_tree_init(ltd_tree* tree, void* d_mem, size_t bytes, int32_t batch,
                         int32_t max_depth, int32_t k, int64_t max_vocab) {
  if (tree == nullptr || d_mem == nullptr) return LTD_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(d_mem) & 255u) != 0) return LTD_ERR_INVALID_ARG;
  const size_t need = ltd_tree_bytes(batch, max_depth, k, max_vocab);
  if (need == 0) return LTD_ERR_SHAPE;
  if (bytes < need) return LTD_ERR_SHAPE;
  const int64_t mn = tree_nodes(max_depth, k);
  const size_t nodes = static_cast<size_t>(batch) * mn;
  char* p = static_cast<char*>(d_mem);
  auto take = [&p](size_t n) {
    char* r = p;
    p += align256(n);
    return r;
  };
  tree->batch = batch;
  tree->max_depth = max_depth;
  tree->k = k;
  tree->max_nodes = static_cast<int32_t>(mn);
  tree->max_vocab = max_vocab;
  tree->token = reinterpret_cast<int32_t*>(take(nodes * 4));
  tree->parent = reinterpret_cast<int32_t*>(take(nodes * 4));
  tree->depth = reinterpret_cast<int32_t*>(take(nodes * 4));
  tree->cum_logprob = reinterpret_cast<float*>(take(nodes * 4));
  tree->xrow = reinterpret_cast<int32_t*>(take(nodes * 4));
  tree->xlse = reinterpret_cast<float*>(take(nodes * 4));
  tree->frontier = reinterpret_cast<int32_t*>(take(static_cast<size_t>(batch) * k * 4));
  tree->n_nodes = reinterpret_cast<int32_t*>(take(static_cast<size_t>(batch) * 4));
  tree->n_levels = reinterpret_cast<int32_t*>(take(static_cast<size_t>(batch) * 4));
  tree->scratch_bytes = expand_scratch_bytes(batch, k, max_vocab);
  tree->scratch = take(tree->scratch_bytes);
  return LTD_OK;
}

ltd_status ltd_tree_reset(const ltd_tree* tree, const int32_t* d_root_tokens,
                          ltd_stream_t stream) {
  const ApiRange nvtx_range("ltd_tree_reset");
  if (!tree_ok(tree) || d_root_tokens == nullptr) return LTD_ERR_INVALID_ARG;
  return from_cuda(launch_tree_reset(tree, d_root_tokens, reinterpret_cast<cudaStream_t>(stream)));
}

ltd_status ltd_expand_tree(const ltd_tree* tree, int32_t level, const void* d_draft_rows,
                           ltd_dtype dtype, int64_t vocab, int64_t rows_per_seq,
                           const int32_t* d_active, ltd_stream_t stream) {
  const ApiRange nvtx_range("ltd_expand_tree");
  if (!tree_ok(tree) || d_draft_rows == nullptr || !dtype_ok(dtype)) return LTD_ERR_INVALID_ARG;
  if (level < 1 || level > tree->max_depth) return LTD_ERR_SHAPE;
  if (vocab < tree->k || vocab > tree->max_vocab) return LTD_ERR_SHAPE;
  if (rows_per_seq < 1 + static_cast<int64_t>(tree->max_depth - 1) * tree->k) return LTD_ERR_SHAPE;
  if (!aligned16(d_draft_rows) || (vocab * static_cast<int64_t>(dtype_size(dtype))) % 16 != 0)
    return LTD_ERR_SHAPE;
  uint32_t* err = device_error_word();
  if (err == nullptr) return LTD_ERR_CUDA;
  const int32_t F = (level == 1) ? 1 : tree->k;
  if (vocab > kExpandMaxVocab) return LTD_ERR_UNSUPPORTED;
  ExpandParams p{};
  p.token = tree->token;
  p.parent = tree->parent;
  p.depth = tree->depth;
  p.cum = tree->cum_logprob;
  p.xrow = tree->xrow;
  p.xlse = tree->xlse;
  p.frontier = tree->frontier;
  p.n_nodes = tree->n_nodes;
  p.n_levels = tree->n_levels;
  p.max_nodes = tree->max_nodes;
  p.k = tree->k;
  p.batch = tree->batch;
  p.rec = static_cast<uint64_t*>(tree->scratch);
  p.rec_chunks = expand_rec_chunks(tree->max_vocab);
  p.rows = d_draft_rows;
  p.vocab = vocab;
  p.rows_per_seq = rows_per_seq;
  p.active = d_active;
  p.level = level;
  p.F = F;
  p.err = err;
  return from_cuda(launch_expand(p, dtype, reinterpret_cast<cudaStream_t>(stream)));
}

ltd_status ltd_depth_observation(const ltd_tree* tree, const int32_t* d_ctx, float* d_out,
                                 ltd_stream_t stream) {
  const ApiRange nvtx_range("ltd_depth_observation");
  if (!tree_ok(tree) || d_ctx == nullptr || d_out == nullptr) return LTD_ERR_INVALID_ARG;
  return from_cuda(launch_depth_obs(tree, d_ctx, d_out, reinterpret_cast<cudaStream_t>(stream)));
}

ltd_status ltd_size_observation(const ltd_tree* tree, const int32_t* d_ctx, int32_t v_pad,
                                float* d_out, ltd_stream_t stream) {
  const ApiRange nvtx_range("ltd_size_observation");
  if (!tree_ok(tree) || d_ctx == nullptr || d_out == nullptr) return LTD_ERR_INVALID_ARG;
  if (v_pad < tree->max_nodes) return LTD_ERR_SHAPE;
  return from_cuda(
      launch_size_obs(tree, d_ctx, v_pad, d_out, reinterpret_cast<cudaStream_t>(stream)));
}

// Common checks of a policy network; n_in is the observation length.
static ltd_status mlp_ok(const ltd_mlp* net, int32_t n_in) {
  if (net == nullptr || net->n_layers < 1 || net->n_layers > LTD_MLP_MAX_LAYERS)
    return LTD_ERR_INVALID_ARG;
  if (net->layout != LTD_MLP_ROW_MAJOR && net->layout != LTD_MLP_PACKED) return LTD_ERR_INVALID_ARG;
  for (int l = 0; l < net->n_layers; ++l)
    if (net->w[l] == nullptr || net->b[l] == nullptr ||
        reinterpret_cast<uintptr_t>(net->w[l]) % 16 != 0)
      return LTD_ERR_INVALID_ARG;
  if (n_in >= 0 && net->dims[0] != n_in) return LTD_ERR_SHAPE;
  if (net->dims[0] < 1) return LTD_ERR_SHAPE;
  for (int l = 1; l <= net->n_layers; ++l)
    if (net->dims[l] < 1 || net->dims[l] > LTD_MLP_MAX_WIDTH) return LTD_ERR_SHAPE;
  return LTD_OK;
}

size_t ltd_mlp_packed_bytes(const ltd_mlp* net) {
  if (mlp_ok(net, -1) != LTD_OK) return 0;
  size_t off[LTD_MLP_MAX_LAYERS];
  return mlp_packed_floats(net, off) * sizeof(float);
}

ltd_status ltd_mlp_pack(const ltd_mlp* net, void* d_mem, size_t bytes, ltd_mlp* packed,
                        ltd_stream_t stream) {
  const ApiRange nvtx_range("ltd_mlp_pack");
  if (packed == nullptr || d_mem == nullptr || reinterpret_cast<uintptr_t>(d_mem) % 256 != 0)
    return LTD_ERR_INVALID_ARG;
  const ltd_status st = mlp_ok(net, -1);
  if (st != LTD_OK) return st;
  if (net->layout != LTD_MLP_ROW_MAJOR) return LTD_ERR_INVALID_ARG;
  if (bytes < ltd_mlp_packed_bytes(net)) return LTD_ERR_SHAPE;
  return from_cuda(launch_mlp_pack(net, static_cast<float*>(d_mem), packed,
                                   reinterpret_cast<cudaStream_t>(stream)));
}

ltd_status ltd_depth_policy(const ltd_tree* tree, const int32_t* d_ctx, const ltd_mlp* net,
                            const int32_t* d_active_in, int32_t* d_active_out, float* d_logits,
                            ltd_stream_t stream) {
  const ApiRange nvtx_range("ltd_depth_policy");
  if (!tree_ok(tree) || d_ctx == nullptr || d_active_out == nullptr) return LTD_ERR_INVALID_ARG;
  const ltd_status st = mlp_ok(net, tree->k * tree->k + 2);
  if (st != LTD_OK) return st;
  if (net->dims[net->n_layers] != 2) return LTD_ERR_SHAPE;
  return from_cuda(launch_mlp_policy(tree, d_ctx, net, 0, 0, d_active_in, d_active_out, 0,
                                     nullptr, d_logits, reinterpret_cast<cudaStream_t>(stream)));
}

ltd_status ltd_size_policy(const ltd_tree* tree, const int32_t* d_ctx, int32_t v_pad,
                           const ltd_mlp* net, int32_t n_cap, int32_t* d_n_verify,
                           float* d_logits, ltd_stream_t stream) {
  const ApiRange nvtx_range("ltd_size_policy");
  if (!tree_ok(tree) || d_ctx == nullptr || d_n_verify == nullptr) return LTD_ERR_INVALID_ARG;
  if (v_pad < tree->max_nodes || v_pad > 8192 || n_cap < 1) return LTD_ERR_SHAPE;
  const ltd_status st = mlp_ok(net, v_pad + 2);
  if (st != LTD_OK) return st;
  return from_cuda(launch_mlp_policy(tree, d_ctx, net, 1, v_pad, nullptr, nullptr, n_cap,
                                     d_n_verify, d_logits, reinterpret_cast<cudaStream_t>(stream)));
}

ltd_status ltd_select_verify(const ltd_tree* tree, const int32_t* d_n_verify, int32_t n_max,
                             const int32_t* d_ctx, int32_t* d_node_ids, int32_t* d_pos,
                             uint32_t* d_mask, ltd_stream_t stream) {
  const ApiRange nvtx_range("ltd_select_verify");
  if (!tree_ok(tree) || !d_n_verify || !d_ctx || !d_node_ids || !d_pos || !d_mask)
    return LTD_ERR_INVALID_ARG;
  if (n_max < 1 || n_max > LTD_MAX_N) return LTD_ERR_SHAPE;
  uint32_t* err = device_error_word();
  if (err == nullptr) return LTD_ERR_CUDA;
  SelectParams p{};
  p.token = tree->token;
  p.parent = tree->parent;
  p.depth = tree->depth;
  p.cum = tree->cum_logprob;
  p.n_nodes = tree->n_nodes;
  p.max_nodes = tree->max_nodes;
  p.n_verify = d_n_verify;
  p.n_max = n_max;
  p.ctx = d_ctx;
  p.node_ids = d_node_ids;
  p.pos = d_pos;
  p.mask = d_mask;
  p.err = err;
  return from_cuda(launch_select(p, tree->batch, reinterpret_cast<cudaStream_t>(stream)));
}

size_t ltd_attention_workspace_bytes(int32_t batch, int32_t hq, int32_t hkv, int32_t head_dim,
                                     int32_t n_max, int32_t max_ctx, ltd_dtype dtype) {
  if (batch < 1 || hq < 1 || hkv < 1 || hq % hkv != 0 || n_max < 1 || max_ctx < 0) return 0;
  AttnParams p{};
  p.batch = batch;
  p.hq = hq;
  p.hkv = hkv;
  p.d = head_dim;
  p.n_max = n_max;
  p.max_ctx = max_ctx;
  size_t ws = 256;  // never zero, so 0 can mean "bad sizes"
  if (attn_tc_supported(p, dtype)) {
    const size_t t = attn_tc_workspace(batch, hq, hkv, head_dim, n_max, max_ctx);
    ws = t > ws ? t : ws;
  }
  return ws;
}

namespace {
ltd_status tree_attention(const void* d_q, const void* d_k, const void* d_v, void* d_out,
                          ltd_dtype dtype, int32_t batch, int32_t hq, int32_t hkv, int32_t head_dim,
                          int32_t s_cap, const int32_t* d_ctx, int32_t max_ctx,
                          const int32_t* d_n_verify, int32_t n_max, const uint32_t* d_mask,
                          float scale, void* d_workspace, size_t workspace_bytes,
                          const void* d_next_k, const void* d_next_v, ltd_stream_t stream) {
  if (!d_q || !d_k || !d_v || !d_out || !d_ctx || !d_n_verify || !d_mask || !dtype_ok(dtype))
    return LTD_ERR_INVALID_ARG;
  if (batch < 1 || hq < 1 || hkv < 1 || hq % hkv != 0 || n_max < 1 || n_max > LTD_MAX_N ||
      max_ctx < 0 || s_cap < 1 || static_cast<int64_t>(max_ctx) + n_max > s_cap)
    return LTD_ERR_SHAPE;
  if (head_dim != 32 && head_dim != 64 && head_dim != 96 && head_dim != 128)
    return LTD_ERR_UNSUPPORTED;
  if (!(scale > 0.f)) return LTD_ERR_INVALID_ARG;
  if (!aligned16(d_q) || !aligned16(d_k) || !aligned16(d_v) || !aligned16(d_out))
    return LTD_ERR_SHAPE;
  if ((d_next_k == nullptr) != (d_next_v == nullptr)) return LTD_ERR_INVALID_ARG;
  if (!aligned16(d_next_k) || !aligned16(d_next_v)) return LTD_ERR_SHAPE;
  const size_t need =
      ltd_attention_workspace_bytes(batch, hq, hkv, head_dim, n_max, max_ctx, dtype);
  if (d_workspace == nullptr || workspace_bytes < need) return LTD_ERR_SHAPE;
  uint32_t* err = device_error_word();
  if (err == nullptr) return LTD_ERR_CUDA;
  AttnParams p{};
  p.q = d_q;
  p.k = d_k;
  p.v = d_v;
  p.out = d_out;
  p.batch = batch;
  p.hq = hq;
  p.hkv = hkv;
  p.d = head_dim;
  p.s_cap = s_cap;
  p.ctx = d_ctx;
  p.max_ctx = max_ctx;
  p.n_verify = d_n_verify;
  p.n_max = n_max;
  p.mask = d_mask;
  p.scale = scale;
  p.ws = d_workspace;
  p.ws_bytes = workspace_bytes;
  p.next_k = d_next_k;
  p.next_v = d_next_v;
  p.err = err;
  const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (attn_tc_supported(p, dtype)) return from_cuda(launch_attn_tc(p, s));
  return from_cuda(launch_attn_simt(p, dtype, s));
}
}  // namespace

ltd_status ltd_tree_attention(const void* d_q, const void* d_k, const void* d_v, void* d_out,
                              ltd_dtype dtype, int32_t batch, int32_t hq, int32_t hkv,
                              int32_t head_dim, int32_t s_cap, const int32_t* d_ctx,
                              int32_t max_ctx, const int32_t* d_n_verify, int32_t n_max,
                              const uint32_t* d_mask, float scale, void* d_workspace,
                              size_t workspace_bytes, ltd_stream_t stream) {
  const ApiRange nvtx_range("ltd_tree_attention");
  return tree_attention(d_q, d_k, d_v, d_out, dtype, batch, hq, hkv, head_dim, s_cap, d_ctx, max_ctx,
                        d_n_verify, n_max, d_mask, scale, d_workspace, workspace_bytes, nullptr,
                        nullptr, stream);
}

ltd_status ltd_tree_attention_next(const void* d_q, const void* d_k, const void* d_v, void* d_out,
                                   ltd_dtype dtype, int32_t batch, int32_t hq, int32_t hkv,
                                   int32_t head_dim, int32_t s_cap, const int32_t* d_ctx,
                                   int32_t max_ctx, const int32_t* d_n_verify, int32_t n_max,
                                   const uint32_t* d_mask, float scale, void* d_workspace,
                                   size_t workspace_bytes, const void* d_next_k,
                                   const void* d_next_v, ltd_stream_t stream) {
  const ApiRange nvtx_range("ltd_tree_attention_next");
  return tree_attention(d_q, d_k, d_v, d_out, dtype, batch, hq, hkv, head_dim, s_cap, d_ctx, max_ctx,
                        d_n_verify, n_max, d_mask, scale, d_workspace, workspace_bytes, d_next_k,
                        d_next_v, stream);
}

int32_t ltd_attention_kernel(ltd_dtype dtype, int32_t batch, int32_t hq, int32_t hkv,
                             int32_t head_dim, int32_t n_max, int32_t max_ctx, int32_t* launches) {
  if (!dtype_ok(dtype) || (head_dim != 32 && head_dim != 64 && head_dim != 96 && head_dim != 128) ||
      batch < 1 || hq < 1 || hkv < 1 || hq % hkv != 0 || n_max < 1 || n_max > LTD_MAX_N ||
      max_ctx < 0)
    return -1;
  AttnParams p{};
  p.batch = batch;
  p.hq = hq;
  p.hkv = hkv;
  p.d = head_dim;
  p.n_max = n_max;
  p.max_ctx = max_ctx;
  const bool tc = attn_tc_supported(p, dtype);
  if (launches) *launches = tc ? attn_tc_launches(batch, hq, hkv, n_max, max_ctx) : 1;
  return tc ? 1 : 0;
}

size_t ltd_lm_head_workspace_bytes(int32_t rows, int64_t vocab, int32_t hidden) {
  if (rows < 1 || rows > LTD_LM_HEAD_MAX_ROWS || vocab < 1 || vocab > 0x7FFFFFFF || hidden < 64 ||
      hidden % 64 != 0)
    return 0;
  return lm_head_workspace(rows, vocab);
}

ltd_status ltd_lm_head_row_stats(const void* d_hidden, const void* d_weight, int32_t rows,
                                 int64_t vocab, int32_t hidden, void* d_logits, float* d_row_max,
                                 float* d_row_lse, int32_t* d_row_argmax, void* d_workspace,
                                 size_t workspace_bytes, ltd_stream_t stream) {
  const ApiRange nvtx_range("ltd_lm_head_row_stats");
  if (!d_hidden || !d_weight || !d_row_max || !d_row_lse || !d_row_argmax || !d_workspace)
    return LTD_ERR_INVALID_ARG;
  const size_t need = ltd_lm_head_workspace_bytes(rows, vocab, hidden);
  if (need == 0 || workspace_bytes < need) return LTD_ERR_SHAPE;
  if (!aligned16(d_hidden) || !aligned16(d_weight) || !aligned16(d_workspace)) return LTD_ERR_SHAPE;
  if (d_logits != nullptr && ((reinterpret_cast<uintptr_t>(d_logits) & 1u) != 0)) return LTD_ERR_SHAPE;
  uint32_t* err = device_error_word();
  if (err == nullptr) return LTD_ERR_CUDA;
  LmHeadParams p{};
  p.hidden_states = d_hidden;
  p.weight = d_weight;
  p.rows = rows;
  p.hidden = hidden;
  p.vocab = vocab;
  p.logits = d_logits;
  p.row_max = d_row_max;
  p.row_lse = d_row_lse;
  p.row_argmax = d_row_argmax;
  p.ws = d_workspace;
  p.ws_bytes = workspace_bytes;
  p.err = err;
  return from_cuda(launch_lm_head(p, reinterpret_cast<cudaStream_t>(stream)));
}

ltd_status ltd_debug_attention_wait(uint64_t limit_ns, uint32_t extra_arrivals) {
  if (extra_arrivals > 1024) return LTD_ERR_INVALID_ARG;
  set_attn_wait_hook(AttnWaitHook{limit_ns, extra_arrivals});
  return LTD_OK;
}

ltd_status ltd_debug_expand_wait(uint64_t limit_ns, uint32_t tag_offset) {
  if (tag_offset > 1024) return LTD_ERR_INVALID_ARG;
  set_expand_wait_hook(ExpandWaitHook{limit_ns, tag_offset});
  return LTD_OK;
}

ltd_status ltd_selftest_umma(int32_t mode, const void* d_a, const void* d_b, float* d_c,
                             ltd_stream_t stream) {
  if ((mode != 0 && mode != 1) || !d_a || !d_b || !d_c) return LTD_ERR_INVALID_ARG;
  if (!aligned16(d_a) || !aligned16(d_b) || !aligned16(d_c)) return LTD_ERR_SHAPE;
  uint32_t* err = device_error_word();
  if (err == nullptr) return LTD_ERR_CUDA;
  return from_cuda(
      launch_umma_selftest(mode, d_a, d_b, d_c, err, reinterpret_cast<cudaStream_t>(stream)));
}

size_t ltd_accept_workspace_bytes(int32_t batch, int32_t n_max, int64_t vocab) {
  if (batch < 1 || n_max < 1 || n_max > LTD_MAX_N || vocab < 1) return 0;
  return accept_workspace(batch, n_max, vocab);
}

ltd_status ltd_kv_append(const ltd_kv_cache* kv, int32_t batch, int32_t n_max,
                         const void* d_new_k, const void* d_new_v, const int32_t* d_ctx,
                         const int32_t* d_n_verify, ltd_stream_t stream) {
  const ApiRange nvtx_range("ltd_kv_append");
  if (kv == nullptr || !kv->d_k_layers || !kv->d_v_layers || !d_new_k || !d_new_v || !d_ctx ||
      !d_n_verify || !dtype_ok(kv->dtype))
    return LTD_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(d_new_k) % 16 != 0 ||
      reinterpret_cast<uintptr_t>(d_new_v) % 16 != 0)
    return LTD_ERR_INVALID_ARG;
  if (batch < 1 || n_max < 1 || n_max > LTD_MAX_N || kv->n_layers < 1 || kv->hkv < 1 ||
      kv->s_cap < 1)
    return LTD_ERR_SHAPE;
  const int64_t row_bytes = static_cast<int64_t>(kv->head_dim) * dtype_size(kv->dtype);
  if (kv->head_dim < 1 || row_bytes % 16 != 0 || row_bytes > 512) return LTD_ERR_UNSUPPORTED;
  uint32_t* err = device_error_word();
  if (err == nullptr) return LTD_ERR_CUDA;
  AppendParams p{};
  p.k_layers = kv->d_k_layers;
  p.v_layers = kv->d_v_layers;
  p.new_k = static_cast<const uint8_t*>(d_new_k);
  p.new_v = static_cast<const uint8_t*>(d_new_v);
  p.n_layers = kv->n_layers;
  p.batch = batch;
  p.hkv = kv->hkv;
  p.s_cap = kv->s_cap;
  p.n_max = n_max;
  p.row_bytes = static_cast<int32_t>(row_bytes);
  p.ctx = d_ctx;
  p.n_verify = d_n_verify;
  p.err = err;
  return from_cuda(launch_append(p, reinterpret_cast<cudaStream_t>(stream)));
}

ltd_status ltd_kv_compact(const ltd_kv_cache* kv, int32_t batch, const int32_t* d_path,
                          int32_t path_stride, const int32_t* d_accept_len, const int32_t* d_ctx,
                          ltd_stream_t stream) {
  const ApiRange nvtx_range("ltd_kv_compact");
  if (kv == nullptr || !kv->d_k_layers || !kv->d_v_layers || !d_path || !d_accept_len || !d_ctx ||
      !dtype_ok(kv->dtype))
    return LTD_ERR_INVALID_ARG;
  if (batch < 1 || kv->n_layers < 1 || kv->hkv < 1 || kv->s_cap < 1 || path_stride < 1)
    return LTD_ERR_SHAPE;
  const int64_t row_bytes = static_cast<int64_t>(kv->head_dim) * dtype_size(kv->dtype);
  if (kv->head_dim < 1 || row_bytes % 16 != 0 || row_bytes > 512) return LTD_ERR_UNSUPPORTED;
  uint32_t* err = device_error_word();
  if (err == nullptr) return LTD_ERR_CUDA;
  CompactParams p{};
  p.k_layers = kv->d_k_layers;
  p.v_layers = kv->d_v_layers;
  p.n_layers = kv->n_layers;
  p.hkv = kv->hkv;
  p.s_cap = kv->s_cap;
  p.row_bytes = static_cast<int32_t>(row_bytes);
  p.path = d_path;
  p.path_stride = path_stride;
  p.accept_len = d_accept_len;
  p.ctx = d_ctx;
  p.err = err;
  return from_cuda(launch_compact(p, batch, reinterpret_cast<cudaStream_t>(stream)));
}

}  // extern "C"

namespace {
ltd_status accept_impl(const ltd_tree* tree, const void* d_target_logits, const void* d_draft_rows,
                       ltd_dtype dtype, int64_t vocab, int64_t rows_per_seq,
                       const int32_t* d_node_ids, const int32_t* d_n_verify, int32_t n_max,
                       const int32_t* d_mode, float temperature, uint64_t seed, uint64_t cycle,
                       const int32_t* d_ctx, int32_t* d_new_ctx, int32_t* d_path,
                       int32_t* d_accept_len, int32_t* d_bonus, const ltd_kv_cache* kv,
                       void* d_workspace, size_t workspace_bytes, ltd_stream_t stream) {
  if (!(temperature > 0.f) || !(temperature <= 3.0e38f)) return LTD_ERR_INVALID_ARG;
  if (!tree_ok(tree) || !d_target_logits || !d_draft_rows || !dtype_ok(dtype) || !d_node_ids ||
      !d_n_verify || !d_mode || !d_ctx || !d_new_ctx || !d_path || !d_accept_len || !d_bonus)
    return LTD_ERR_INVALID_ARG;
  if (n_max < 1 || n_max > LTD_MAX_N || vocab < 1 || vocab > tree->max_vocab) return LTD_ERR_SHAPE;
  if (rows_per_seq < 1 + static_cast<int64_t>(tree->max_depth - 1) * tree->k) return LTD_ERR_SHAPE;
  if (!aligned16(d_target_logits) || (vocab * static_cast<int64_t>(dtype_size(dtype))) % 16 != 0)
    return LTD_ERR_SHAPE;
  if (vocab > kAcceptMaxVocab) return LTD_ERR_UNSUPPORTED;
  const size_t need = accept_workspace(tree->batch, n_max, vocab);
  if (d_workspace == nullptr || workspace_bytes < need) return LTD_ERR_SHAPE;
  if (kv != nullptr) {
    if (!kv->d_k_layers || !kv->d_v_layers || !dtype_ok(kv->dtype)) return LTD_ERR_INVALID_ARG;
    const int64_t row_bytes = static_cast<int64_t>(kv->head_dim) * dtype_size(kv->dtype);
    if (kv->n_layers < 1 || kv->hkv < 1 || kv->s_cap < 1) return LTD_ERR_SHAPE;
    if (kv->head_dim < 1 || row_bytes % 16 != 0 || row_bytes > 512) return LTD_ERR_UNSUPPORTED;
  }
  uint32_t* err = device_error_word();
  if (err == nullptr) return LTD_ERR_CUDA;
  AcceptParams p{};
  p.token = tree->token;
  p.parent = tree->parent;
  p.xrow = tree->xrow;
  p.xlse = tree->xlse;
  p.max_nodes = tree->max_nodes;
  p.max_depth = tree->max_depth;
  p.target = d_target_logits;
  p.draft = d_draft_rows;
  p.vocab = vocab;
  p.rows_per_seq = rows_per_seq;
  p.node_ids = d_node_ids;
  p.n_verify = d_n_verify;
  p.n_max = n_max;
  p.mode = d_mode;
  p.seed = seed;
  p.cycle = cycle;
  p.ctx = d_ctx;
  p.new_ctx = d_new_ctx;
  p.path = d_path;
  p.accept_len = d_accept_len;
  p.bonus = d_bonus;
  p.rec = static_cast<AcceptRecord*>(d_workspace);
  p.inv_t = temperature == 1.f ? 1.f : 1.f / temperature;
  p.tempered = temperature != 1.f;
  p.err = err;
  const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e = launch_accept(p, tree->batch, dtype, s);
  if (e != cudaSuccess || kv == nullptr) return from_cuda(e);
  return ltd_kv_compact(kv, tree->batch, d_path, tree->max_depth + 1, d_accept_len, d_ctx, stream);
}
}  // namespace

extern "C" {

ltd_status ltd_accept(const ltd_tree* tree, const void* d_target_logits, const void* d_draft_rows,
                      ltd_dtype dtype, int64_t vocab, int64_t rows_per_seq,
                      const int32_t* d_node_ids, const int32_t* d_n_verify, int32_t n_max,
                      const int32_t* d_mode, uint64_t seed, uint64_t cycle, const int32_t* d_ctx,
                      int32_t* d_new_ctx, int32_t* d_path, int32_t* d_accept_len,
                      int32_t* d_bonus, const ltd_kv_cache* kv, void* d_workspace,
                      size_t workspace_bytes, ltd_stream_t stream) {
  const ApiRange nvtx_range("ltd_accept");
  return accept_impl(tree, d_target_logits, d_draft_rows, dtype, vocab, rows_per_seq, d_node_ids,
                     d_n_verify, n_max, d_mode, 1.f, seed, cycle, d_ctx, d_new_ctx, d_path,
                     d_accept_len, d_bonus, kv, d_workspace, workspace_bytes, stream);
}

ltd_status ltd_accept_tempered(const ltd_tree* tree, const void* d_target_logits,
                               const void* d_draft_rows, ltd_dtype dtype, int64_t vocab,
                               int64_t rows_per_seq, const int32_t* d_node_ids,
                               const int32_t* d_n_verify, int32_t n_max, const int32_t* d_mode,
                               float temperature, uint64_t seed, uint64_t cycle,
                               const int32_t* d_ctx, int32_t* d_new_ctx, int32_t* d_path,
                               int32_t* d_accept_len, int32_t* d_bonus, const ltd_kv_cache* kv,
                               void* d_workspace, size_t workspace_bytes, ltd_stream_t stream) {
  const ApiRange nvtx_range("ltd_accept_tempered");
  return accept_impl(tree, d_target_logits, d_draft_rows, dtype, vocab, rows_per_seq, d_node_ids,
                     d_n_verify, n_max, d_mode, temperature, seed, cycle, d_ctx, d_new_ctx, d_path,
                     d_accept_len, d_bonus, kv, d_workspace, workspace_bytes, stream);
}

ltd_status ltd_check(ltd_stream_t stream, uint32_t* out_bits) {
  const cudaError_t e = cudaStreamSynchronize(reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return LTD_ERR_CUDA;
  uint32_t* w = device_error_word();
  if (w == nullptr) return LTD_ERR_CUDA;
  uint32_t bits = 0;
  if (cudaMemcpy(&bits, w, sizeof(bits), cudaMemcpyDeviceToHost) != cudaSuccess) return LTD_ERR_CUDA;
  if (bits != 0) {
    const uint32_t zero = 0;
    if (cudaMemcpy(w, &zero, sizeof(zero), cudaMemcpyHostToDevice) != cudaSuccess)
      return LTD_ERR_CUDA;
  }
  if (out_bits) *out_bits = bits;
  if (bits & LTD_DEVERR_TIMEOUT) return LTD_ERR_TIMEOUT;
  if (bits) return LTD_ERR_DEVICE;
  return LTD_OK;
}

}  // extern "C"
