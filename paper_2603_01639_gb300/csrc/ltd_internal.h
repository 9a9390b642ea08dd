// Internal launch interfaces between the C ABI glue (ltd_api.cu) and the
// kernel translation units.  Not part of the public ABI.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "ltd.h"

namespace ltd {

// Address of this device's error word (lives in ltd_api.cu).
uint32_t* device_error_word();

// Whether `t` is a tree that ltd_tree_init carved: sizes within the limits
// and every array present (lives in ltd_api.cu).
bool tree_valid(const ltd_tree* t);

// Whether launches carry the programmatic-dependent-launch attribute (on
// unless the environment sets LTD_NO_PDL=1; read once).
bool pdl_enabled();

// Launch `kernel` with up to three extra launch attributes plus, when
// enabled, programmatic stream serialization (the kernel calls grid_wait()
// before reading another kernel's output).  If the runtime refuses the
// combination, the launch is repeated without it.
template <typename... KArgs, typename... Args>
cudaError_t launch(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                   const cudaLaunchAttribute* extra, int n_extra, Args&&... args) {
  cudaLaunchAttribute attr[4];
  int n = 0;
  for (int i = 0; i < n_extra && i < 3; ++i) attr[n++] = extra[i];
  const int base_n = n;
  if (pdl_enabled()) {
    attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[n].val.programmaticStreamSerializationAllowed = 1;
    ++n;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = n;
  cudaError_t e = cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
  if (e != cudaSuccess && n != base_n) {
    (void)cudaGetLastError();
    cfg.numAttrs = base_n;
    e = cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
  }
  return e;
}

// Work split of a vocabulary scan: `chunks` CTAs per row, each covering
// `chunk_elems` elements (a multiple of 8, so chunk starts stay 16-byte
// aligned for both dtypes).
struct VocabSplit {
  int32_t chunks;
  int64_t chunk_elems;
};
VocabSplit vocab_split(int64_t rows, int64_t vocab, int64_t target_ctas, int64_t min_elems);

// ------------------------------------------------------------- expansion
// A draft row is cut into items of 16 KB (8192 bf16 or 4096 fp32 entries);
// each item's record (its top-k keys and its (max, sum of exp), every
// 64-bit word tagged with the level) goes to the tree's scratch area, laid
// out [batch][k rows][rec_chunks][k + 2 words].
constexpr int64_t kExpandMaxVocab = int64_t(1) << 20;
int32_t expand_rec_chunks(int64_t max_vocab);
size_t expand_scratch_bytes(int32_t batch, int32_t k, int64_t max_vocab);

struct ExpandParams {
  int32_t* token;
  int32_t* parent;
  int32_t* depth;
  float* cum;
  int32_t* xrow;
  float* xlse;
  int32_t* frontier;
  int32_t* n_nodes;
  int32_t* n_levels;
  int32_t max_nodes;
  int32_t k;
  int32_t batch;
  uint64_t* rec;       // the tree's scratch area
  int32_t rec_chunks;  // items per row the records are laid out for
  const void* rows;
  int64_t vocab;
  int64_t rows_per_seq;
  const int32_t* active;
  int32_t level;
  int32_t F;              // rows per sequence at this level
  int32_t item_elems;     // entries per item (set by launch_expand)
  int32_t chunks;         // items per row (set by launch_expand)
  int32_t n_items;        // batch * F * chunks (set by launch_expand)
  int32_t items_per_cta;  // (set by the launch)
  uint64_t wait_limit_ns; // consumer's wait on the records (set by launch_expand)
  uint32_t tag_offset;    // added to the tag the consumer waits for (test hook)
  int32_t j_row;          // leading keys per item list for the row threshold (set by launch_expand)
  uint32_t* err;
};
// Test hook of the expansion consumer's wait (k_expand.cu): its limit (0 =
// the default 1 s) and an offset to the awaited tag that no producer writes.
struct ExpandWaitHook {
  uint64_t limit_ns;
  uint32_t tag_offset;
};
void set_expand_wait_hook(const ExpandWaitHook& h);
cudaError_t launch_tree_reset(const ltd_tree* t, const int32_t* roots, cudaStream_t s);
cudaError_t launch_expand(const ExpandParams& p, ltd_dtype dtype, cudaStream_t s);

// ------------------------------------------------------------- selection
struct SelectParams {
  const int32_t* token;
  const int32_t* parent;
  const int32_t* depth;
  const float* cum;
  const int32_t* n_nodes;
  int32_t max_nodes;
  const int32_t* n_verify;
  int32_t n_max;
  const int32_t* ctx;
  int32_t* node_ids;
  int32_t* pos;
  uint32_t* mask;
  uint32_t* err;
};
cudaError_t launch_select(const SelectParams& p, int32_t batch, cudaStream_t s);

// ------------------------------------------------------------- attention
struct AttnParams {
  const void* q;
  const void* k;
  const void* v;
  void* out;
  int32_t batch, hq, hkv, d, s_cap;
  const int32_t* ctx;
  int32_t max_ctx;
  const int32_t* n_verify;
  int32_t n_max;
  const uint32_t* mask;
  float scale;
  void* ws;
  size_t ws_bytes;
  const void* next_k;  // L2 prefetch hint for the next call (may be null)
  const void* next_v;
  uint32_t* err;
};
size_t attn_simt_workspace(const AttnParams& p);
cudaError_t launch_attn_simt(const AttnParams& p, ltd_dtype dtype, cudaStream_t s);
bool attn_tc_supported(const AttnParams& p, ltd_dtype dtype);
// Streaming multiprocessors of the current device (152 if it cannot be asked).
int device_sm_count();
// Test hook of the tensor-core kernel's split-counter wait (k_attn_tc.cu):
// its limit (0 = the default 1 s) and arrivals awaited beyond the splits.
struct AttnWaitHook {
  uint64_t limit_ns;
  uint32_t extra_arrivals;
};
void set_attn_wait_hook(const AttnWaitHook& h);
AttnWaitHook attn_wait_hook();
size_t attn_tc_workspace(int32_t batch, int32_t hq, int32_t hkv, int32_t d, int32_t n_max,
                         int32_t max_ctx);
cudaError_t launch_attn_tc(const AttnParams& p, cudaStream_t s);
int32_t attn_tc_launches(int32_t batch, int32_t hq, int32_t hkv, int32_t n_max,
                         int32_t max_ctx);
cudaError_t launch_umma_selftest(int mode, const void* a, const void* b, float* c, uint32_t* err,
                                 cudaStream_t s);

// ------------------------------------------------------------- LM head
struct LmHeadParams {
  const void* hidden_states;  // [rows][hidden] bf16
  const void* weight;         // [vocab][hidden] bf16
  int32_t rows, hidden;
  int64_t vocab;
  void* logits;               // [rows][vocab] bf16 or null
  float* row_max;
  float* row_lse;
  int32_t* row_argmax;
  void* ws;
  size_t ws_bytes;
  uint32_t* err;
};
size_t lm_head_workspace(int32_t rows, int64_t vocab);
cudaError_t launch_lm_head(const LmHeadParams& p, cudaStream_t s);

// ------------------------------------------------------------- acceptance
constexpr int64_t kAcceptTargetCtas = 608;
constexpr int64_t kAcceptMinElems = 4096;

// Largest vocabulary the acceptance walk holds in one cluster's shared memory
// (16 CTAs x 16384 fp32 entries of p and q each).
constexpr int64_t kAcceptMaxVocab = 16 * 16384;
struct AcceptRecord {
  float m, s;
  unsigned long long key;
};

struct AcceptParams {
  const int32_t* token;
  const int32_t* parent;
  const int32_t* xrow;
  const float* xlse;
  int32_t max_nodes;
  int32_t max_depth;
  const void* target;
  const void* draft;
  int64_t vocab;
  int64_t rows_per_seq;
  const int32_t* node_ids;
  const int32_t* n_verify;
  int32_t n_max;
  const int32_t* mode;
  unsigned long long seed, cycle;
  const int32_t* ctx;
  int32_t* new_ctx;
  int32_t* path;
  int32_t* accept_len;
  int32_t* bonus;
  AcceptRecord* rec;  // [batch][n_max][chunks]
  float inv_t;        // 1 / temperature of the stochastic rules (1 at T = 1)
  int32_t tempered;   // T != 1: the draft rows' normaliser is computed in the walk
  int32_t chunks;         // units per row (set by the launch)
  int64_t chunk_elems;    // entries per unit (set by the launch)
  int32_t n_units;        // batch * n_max * chunks (set by the launch)
  uint32_t* err;
};
size_t accept_workspace(int32_t batch, int32_t n_max, int64_t vocab);

// Policy observations (k_policy.cu); entries past the tree hold kPolicyPad.
constexpr float kPolicyPad = LTD_POLICY_PAD;
cudaError_t launch_depth_obs(const ltd_tree* t, const int32_t* ctx, float* out, cudaStream_t s);
cudaError_t launch_size_obs(const ltd_tree* t, const int32_t* ctx, int32_t v_pad, float* out,
                            cudaStream_t s);
// Packed policy weights (k_policy.cu): units of a layer's column slice per
// CTA, the packed float count (and each matrix's offset), and the packing.
int mlp_packed_units(int n_out);
size_t mlp_packed_floats(const ltd_mlp* net, size_t offsets[LTD_MLP_MAX_LAYERS]);
cudaError_t launch_mlp_pack(const ltd_mlp* net, float* base, ltd_mlp* packed, cudaStream_t s);
// Depth (size_policy 0) or size (1) policy MLP on the device (k_policy.cu).
cudaError_t launch_mlp_policy(const ltd_tree* t, const int32_t* ctx, const ltd_mlp* net,
                              int32_t size_policy, int32_t v_pad, const int32_t* active_in,
                              int32_t* active_out, int32_t n_cap, int32_t* n_verify,
                              float* logits, cudaStream_t s);
cudaError_t launch_accept(const AcceptParams& p, int32_t batch, ltd_dtype dtype, cudaStream_t s);

struct CompactParams {
  void* const* k_layers;
  void* const* v_layers;
  int32_t n_layers, hkv, s_cap;
  int32_t row_bytes;
  const int32_t* path;
  int32_t path_stride;
  const int32_t* accept_len;
  const int32_t* ctx;
  uint32_t* err;
};
cudaError_t launch_compact(const CompactParams& p, int32_t batch, cudaStream_t s);

// The verified tokens' new K/V rows into every layer's cache (k_accept.cu).
struct AppendParams {
  void* const* k_layers;
  void* const* v_layers;
  const uint8_t* new_k;  // [n_layers][batch][hkv][n_max][row]
  const uint8_t* new_v;
  int32_t n_layers, batch, hkv, s_cap, n_max;
  int32_t row_bytes;
  const int32_t* ctx;
  const int32_t* n_verify;
  uint32_t* err;
};
cudaError_t launch_append(const AppendParams& p, cudaStream_t s);

}  // namespace ltd
