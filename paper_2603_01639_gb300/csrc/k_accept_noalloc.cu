// ltd_accept_noalloc: the acceptance step without a caller-provided
// workspace.
//
// Some callers cannot allocate device memory at the point where they accept
// a draft: a serving loop that reserved all of its device memory up front
// and forbids allocation on the hot path, a plugin whose host framework owns
// every device buffer, or code that must stay free of allocator calls so a
// stream can later be captured into a CUDA graph with a fixed memory plan.
// For them this entry point keeps the acceptance kernel's scratch (one
// record per slot and vocabulary chunk) in the file-scope array below,
// which every GPU that loads the library holds until the process exits.
//
// Every call shares that one array: two calls whose kernels overlap on the
// GPU (different streams, or a second call before the first finished on a
// different device queue) race on it.  Calls on one stream are ordered and
// safe.
#include <mutex>

#include "ltd_common.cuh"
#include "ltd_internal.h"

namespace ltd {

namespace {

static __device__ __align__(256) unsigned char g_accept_scratch[LTD_ACCEPT_NOALLOC_SCRATCH_BYTES];

// Device address of g_accept_scratch on the current device.  The array's
// name is only a host-side stand-in in host code, so the address comes from
// cudaGetSymbolAddress, once per device, with that device current.
unsigned char* scratch_address() {
  static std::mutex mu;
  static unsigned char* ptrs[128] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 128) return nullptr;
  std::lock_guard<std::mutex> lock(mu);
  if (ptrs[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_accept_scratch) != cudaSuccess) return nullptr;
    ptrs[dev] = static_cast<unsigned char*>(p);
  }
  return ptrs[dev];
}

}  // namespace

}  // namespace ltd

using namespace ltd;

extern "C" ltd_status ltd_accept_noalloc(const ltd_tree* tree, const void* d_target_logits,
                                         const void* d_draft_rows, ltd_dtype dtype, int64_t vocab,
                                         int64_t rows_per_seq, const int32_t* d_node_ids,
                                         const int32_t* d_n_verify, int32_t n_max,
                                         const int32_t* d_mode, uint64_t seed, uint64_t cycle,
                                         const int32_t* d_ctx, int32_t* d_new_ctx, int32_t* d_path,
                                         int32_t* d_accept_len, int32_t* d_bonus,
                                         const ltd_kv_cache* kv, ltd_stream_t stream) {
  // The same argument checks, in the same order, as ltd_accept: a missing or
  // malformed tree or a missing buffer is LTD_ERR_INVALID_ARG before any
  // size is looked at.
  if (!tree_valid(tree) || !d_target_logits || !d_draft_rows || !d_node_ids || !d_n_verify ||
      !d_mode || !d_ctx || !d_new_ctx || !d_path || !d_accept_len || !d_bonus)
    return LTD_ERR_INVALID_ARG;
  if (n_max < 1 || n_max > LTD_MAX_N || vocab < 1) return LTD_ERR_SHAPE;
  const size_t need = ltd_accept_workspace_bytes(tree->batch, n_max, vocab);
  if (need == 0 || need > LTD_ACCEPT_NOALLOC_SCRATCH_BYTES) return LTD_ERR_SHAPE;
  unsigned char* scratch = scratch_address();
  if (scratch == nullptr) return LTD_ERR_CUDA;
  return ltd_accept(tree, d_target_logits, d_draft_rows, dtype, vocab, rows_per_seq, d_node_ids,
                    d_n_verify, n_max, d_mode, seed, cycle, d_ctx, d_new_ctx, d_path, d_accept_len,
                    d_bonus, kv, scratch, LTD_ACCEPT_NOALLOC_SCRATCH_BYTES, stream);
}
