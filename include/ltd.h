/*
 * ltd.h -- C ABI of the GB300 (sm_103a) hot path of one draft-and-verify
 * cycle of "Learning To Draft" (Zhang et al., LTD), section 3.2
 * "Draft-and-Verify Cycle": draft tree generation, candidate token
 * selection, tree-attention verification and acceptance.
 *
 * Conventions shared by every call
 * --------------------------------
 *  - Every pointer named d_* is DEVICE memory owned by the caller.  The
 *    library never allocates, frees or retains caller memory; the only
 *    device memory it owns is one 4-byte error word per device.
 *  - Every call is asynchronous on the given stream and never synchronises,
 *    except ltd_check().  Arguments are validated on the host before any
 *    launch; a bad argument returns an error status and launches nothing.
 *  - Problems only the device can see (a sequence whose per-sequence size
 *    breaks a bound, a bounded wait that gave up) set bits in the device
 *    error word; the kernel skips the offending work and returns.  No kernel
 *    traps or aborts.  ltd_check() synchronises the stream, reads and clears
 *    the word, and maps it to a status.
 *  - Tensors are dense, row-major, innermost dimension last.  Integers are
 *    int32; bit masks are uint32 words, bit j of a row in word j/32 at bit
 *    j%32.  Floating inputs are LTD_F32 or LTD_BF16 as stated per call.
 *  - Batch entries are independent sequences ("b").  Sizes that may differ
 *    per sequence (context, verify size, mode) are device arrays [batch].
 *
 * Readings of the paper (it leaves these open):
 *  - depth L counts the levels below the root, so a tree of L levels holds
 *    V_all = 1 + k + (L-1) k^2 nodes (the paper's formula with D = L + 1);
 *  - the verify size N counts the root, which always occupies slot 0;
 *  - ties break toward the lower token id within a row and toward the lower
 *    node id across nodes.
 */
#ifndef LTD_H
#define LTD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* cudaStream_t without pulling in the CUDA headers. */
typedef struct CUstream_st* ltd_stream_t;

typedef enum ltd_status {
  LTD_OK = 0,
  LTD_ERR_INVALID_ARG = 1, /* null pointer, bad enum, non-positive size   */
  LTD_ERR_SHAPE = 2,       /* sizes inconsistent with each other/limits   */
  LTD_ERR_UNSUPPORTED = 3, /* valid request the library does not implement */
  LTD_ERR_CUDA = 4,        /* a CUDA runtime call failed                  */
  LTD_ERR_DEVICE = 5,      /* a kernel flagged bad per-sequence data      */
  LTD_ERR_TIMEOUT = 6      /* a bounded device wait gave up               */
} ltd_status;

typedef enum ltd_dtype { LTD_F32 = 0, LTD_BF16 = 1 } ltd_dtype;
typedef enum ltd_mode {
  LTD_GREEDY = 0,
  LTD_STOCHASTIC = 1,
  LTD_STOCHASTIC_POINT_MASS = 2,
  LTD_STOCHASTIC_NO_REPLACEMENT = 3
} ltd_mode;

/* Limits of the library. */
#define LTD_MAX_K 32          /* beam width k                              */
#define LTD_MAX_DEPTH 16      /* levels below the root                     */
#define LTD_MAX_N 256         /* verify size, root included               */
#define LTD_MAX_TREE_NODES 4096

/* Device error word bits (ltd_check folds them into one status). */
#define LTD_DEVERR_LEVEL 0x1u     /* expand called out of level order    */
#define LTD_DEVERR_NVERIFY 0x2u   /* N < 1, N > tree size or N > n_max   */
#define LTD_DEVERR_CTX 0x4u       /* ctx < 0, ctx > max_ctx, ctx+N > s_cap */
#define LTD_DEVERR_TREE 0x8u      /* selection not ancestor-closed        */
#define LTD_DEVERR_TIMEOUT 0x10u  /* a bounded wait gave up               */
#define LTD_DEVERR_MODE 0x20u     /* mode not one of ltd_mode             */

/* ------------------------------------------------------------------------
 * Draft tree (section 3.2, "Draft Tree Generation").
 *
 * Structure-of-arrays state of `batch` trees, carved by ltd_tree_init() out
 * of ONE caller-owned device buffer of ltd_tree_bytes() bytes.  Node ids are
 * assigned in expansion order: the root is id 0; level 1 gives ids 1..k in
 * rank order; level l >= 2 gives the child of rank c of the frontier node of
 * rank r the id 1 + k + (l-2) k^2 + r k + c.  All arrays are [batch][...]:
 *   token[max_nodes]        token id of the node
 *   parent[max_nodes]       parent node id, -1 for the root
 *   depth[max_nodes]        0 for the root
 *   cum_logprob[max_nodes]  float, sum of log p along the root->node path
 *   xrow[max_nodes]         draft row that expanded the node, -1 if none
 *   xlse[max_nodes]         float, log-sum-exp of that row
 *   frontier[k]             frontier node ids in rank order
 *   n_nodes[1], n_levels[1] node count and levels built so far
 * The scratch area holds ltd_expand_tree's per-item records (each 64-bit
 * word tagged with the level that wrote it); ltd_tree_reset zeroes it.
 * ------------------------------------------------------------------------ */
typedef struct ltd_tree {
  int32_t batch, max_depth, k, max_nodes;
  int64_t max_vocab;
  int32_t* token;
  int32_t* parent;
  int32_t* depth;
  float* cum_logprob;
  int32_t* xrow;
  float* xlse;
  int32_t* frontier;
  int32_t* n_nodes;
  int32_t* n_levels;
  void* scratch;
  size_t scratch_bytes;
} ltd_tree;

/* Bytes of device memory a tree of these dimensions needs (0 on bad sizes:
 * batch >= 1, 1 <= max_depth <= LTD_MAX_DEPTH, 1 <= k <= LTD_MAX_K,
 * 1 + k + (max_depth-1) k^2 <= LTD_MAX_TREE_NODES, k <= max_vocab). */
size_t ltd_tree_bytes(int32_t batch, int32_t max_depth, int32_t k, int64_t max_vocab);

/* Fill *tree with views into d_mem (host-side pointer arithmetic only; no
 * CUDA call).  d_mem must be 256-byte aligned and hold ltd_tree_bytes(). */
ltd_status ltd_tree_init(ltd_tree* tree, void* d_mem, size_t bytes, int32_t batch,
                         int32_t max_depth, int32_t k, int64_t max_vocab);

/* Start a new cycle: every tree becomes the single root node holding
 * d_root_tokens[b] (the target's bonus token of the previous cycle, section
 * 3.2 "Draft Tree Verification"), and the scratch area is zeroed. */
ltd_status ltd_tree_reset(const ltd_tree* tree, const int32_t* d_root_tokens, ltd_stream_t stream);

/* Expand every active tree by one level (section 3.2, "Draft Tree
 * Generation"): level 1 takes the top-k tokens of the root's row; level
 * l >= 2 gives each of the k frontier nodes its top-k tokens as children
 * (a k^2 pool, all kept) and makes the k children with the largest
 * cumulative log-probability the new frontier.
 *
 *  level           1-based level being built; all active sequences must have
 *                  exactly level-1 levels (else LTD_DEVERR_LEVEL)
 *  d_draft_rows    draft logits [batch][rows_per_seq][vocab] (dtype): row 0
 *                  is the root's distribution, row 1+(l-2)k+r that of the
 *                  frontier node of rank r at level l-1 (read for level l)
 *  rows_per_seq    >= 1 + (max_depth-1) k
 *  d_active        [batch] 0/1, NULL = all sequences expand
 * Per node: cum = cum(parent) + x - logsumexp(row), computed in fp32.
 * Rows must start 16-byte aligned (vocab * sizeof(dtype) % 16 == 0).
 * vocab <= 1,048,576 (larger returns LTD_ERR_UNSUPPORTED).  The records of
 * a level's rows are merged by one CTA per sequence after a bounded wait;
 * if it runs out, LTD_DEVERR_TIMEOUT is flagged and the level stays
 * unbuilt (n_levels unchanged). */
ltd_status ltd_expand_tree(const ltd_tree* tree, int32_t level, const void* d_draft_rows,
                           ltd_dtype dtype, int64_t vocab, int64_t rows_per_seq,
                           const int32_t* d_active, ltd_stream_t stream);

/* Candidate token selection (section 3.2): the N-1 non-root nodes with the
 * largest cum_logprob (ties to the lower id) plus the root, flattened in
 * ascending id order ("slots"), with positions and the tree attention mask.
 *  d_n_verify  [batch] N_b, 1 <= N_b <= min(n_max, n_nodes[b])
 *  d_ctx       [batch] context length before the cycle
 *  d_node_ids  out [batch][n_max]   node id per slot, -1 past N_b
 *  d_pos       out [batch][n_max]   ctx + depth, -1 past N_b
 *  d_mask      out [batch][n_max][ceil(n_max/32)]  bit j of row i set iff
 *              slot j is an ancestor of slot i or i itself; zero past N_b. */
ltd_status ltd_select_verify(const ltd_tree* tree, const int32_t* d_n_verify, int32_t n_max,
                             const int32_t* d_ctx, int32_t* d_node_ids, int32_t* d_pos,
                             uint32_t* d_mask, ltd_stream_t stream);

/* Observations of the learned policies (section 3.1 and Appendix A,
 * "Observation Space"), gathered on the device for a host-side policy.
 * Depth policy, after an expansion:
 *  d_out  [batch][k*k + 2] float: the cum_logprob of the candidate tokens of
 *         the last level built (its k^2 nodes in id order; k at level 1),
 *         padded with LTD_POLICY_PAD to k^2, then the draft depth D (levels
 *         built) and the sequence length L = ctx[b].
 * Size policy, after the draft:
 *  v_pad  >= the tree's max_nodes (1 + k + (max_depth-1) k^2)
 *  d_out  [batch][v_pad + 2] float: the cum_logprob of every node in id
 *         order (root = 0), padded with LTD_POLICY_PAD, then D and L.
 *  d_ctx  [batch] context length.
 * Both only read the tree; the buffers are the caller's. */
#define LTD_POLICY_PAD (-100.0f)
ltd_status ltd_depth_observation(const ltd_tree* tree, const int32_t* d_ctx, float* d_out,
                                 ltd_stream_t stream);
ltd_status ltd_size_observation(const ltd_tree* tree, const int32_t* d_ctx, int32_t v_pad,
                                float* d_out, ltd_stream_t stream);

/* The two policies evaluated on the device, so that a decision needs no
 * round trip to the host and the whole adaptive cycle stays one stream of
 * launches (capturable in one CUDA graph).  A policy is a ReLU MLP (section
 * 3.1; Appendix A.2: the depth policy one hidden layer of 1024 units and two
 * actions STOP = 0 / CONTINUE = 1, the size policy hidden layers of 1024 and
 * 256 units and 12 actions mapped to V = 20, 40, ..., 240):
 *   h_0 = observation (the vectors ltd_depth_observation /
 *         ltd_size_observation write), h_{l+1} = relu(h_l W_l + b_l),
 *   logits = h_{n-1} W_{n-1} + b_{n-1}, action = argmax (ties to the lower
 *   action), all in fp32 (accumulation order fixed, run to run identical).
 * ltd_mlp describes the network; every pointer is device memory owned by
 * the caller and only read:
 *   n_layers   1..LTD_MLP_MAX_LAYERS weight matrices
 *   layout     LTD_MLP_ROW_MAJOR, or LTD_MLP_PACKED for a network that
 *              ltd_mlp_pack() rearranged (the policies then stream each
 *              CTA's weight slice with a few large bulk copies; row-major
 *              weights are read with plain loads, correct but slower)
 *   dims       dims[0] inputs (k^2 + 2 for the depth policy, v_pad + 2 for
 *              the size policy, v_pad <= 8192), dims[n_layers] actions,
 *              hidden widths dims[1..n_layers-1]; every width after dims[0]
 *              in 1..LTD_MLP_MAX_WIDTH
 *   w[l]       [dims[l]][dims[l+1]] float, row-major (h_l W_l), 16-byte
 *              aligned
 *   b[l]       [dims[l+1]] float
 * ltd_depth_policy, after level D of the draft:
 *   d_active_in   [batch] int32, nonzero = the sequence is still drafting
 *                 (NULL = all); d_active_out [batch] int32 (may equal
 *                 d_active_in): 1 where the sequence was active, the policy
 *                 chose CONTINUE and the tree has a level left, else 0.
 *                 Pass d_active_out as the next ltd_expand_tree's d_active.
 *   d_logits      optional [batch][2] float (NULL = not written); rows of
 *                 inactive sequences are written too.
 *   dims[n_layers] must be 2.
 * ltd_size_policy, after the draft:
 *   n_cap         the verify-buffer capacity (n_max of ltd_select_verify)
 *   d_n_verify    [batch] int32 out: N = min(1 + V, n_cap, nodes in the
 *                 tree), V = 20 + 20 a for action a (N counts the root).
 *   d_logits      optional [batch][dims[n_layers]] float.
 *   dims[n_layers] in 1..LTD_MLP_MAX_WIDTH (12 for the paper's policy).
 * Errors: LTD_ERR_INVALID_ARG for NULL tree / d_ctx / net / outputs,
 * n_layers or layout out of range, or weights not 16-byte aligned; LTD_ERR_SHAPE when dims[0] does not match the
 * observation length, a width is out of range, the depth policy does not
 * have 2 actions, or (size policy) v_pad is below the tree's max_nodes or
 * above 8192 or n_cap < 1. */
#define LTD_MLP_MAX_LAYERS 4
#define LTD_MLP_MAX_WIDTH 2048
#define LTD_MLP_ROW_MAJOR 0
#define LTD_MLP_PACKED 1
typedef struct ltd_mlp {
  int32_t n_layers;
  int32_t layout;
  int32_t dims[LTD_MLP_MAX_LAYERS + 1];
  const float* w[LTD_MLP_MAX_LAYERS];
  const float* b[LTD_MLP_MAX_LAYERS];
} ltd_mlp;
/* Rearrange a row-major network for the device policies: each weight
 * matrix is stored as the column slices the policy kernel's CTAs own, each
 * slice [dims[l]][slice width] contiguous and zero-padded to a multiple of
 * four columns.  The layout is private to this library build.
 *  ltd_mlp_packed_bytes  bytes of device memory the packed weights need
 *                        (0 for a network the policies would reject)
 *  ltd_mlp_pack          reads net (LTD_MLP_ROW_MAJOR) on the stream and
 *                        writes the packed weights into d_mem (256-byte
 *                        aligned, >= ltd_mlp_packed_bytes); fills *packed
 *                        with pointers into d_mem, the same dims, the same
 *                        bias pointers and layout LTD_MLP_PACKED. */
size_t ltd_mlp_packed_bytes(const ltd_mlp* net);
ltd_status ltd_mlp_pack(const ltd_mlp* net, void* d_mem, size_t bytes, ltd_mlp* packed,
                        ltd_stream_t stream);
ltd_status ltd_depth_policy(const ltd_tree* tree, const int32_t* d_ctx, const ltd_mlp* net,
                            const int32_t* d_active_in, int32_t* d_active_out, float* d_logits,
                            ltd_stream_t stream);
ltd_status ltd_size_policy(const ltd_tree* tree, const int32_t* d_ctx, int32_t v_pad,
                           const ltd_mlp* net, int32_t n_cap, int32_t* d_n_verify,
                           float* d_logits, ltd_stream_t stream);

/* Tree attention of the verified tokens against the KV cache (section 3.2
 * "Draft Tree Verification"; tree attention as in SpecInfer, section 2.1).
 * For slot i < N_b and query head h, KV head g = h / (hq/hkv):
 *   out[b][i][h] = sum_k softmax_k(scale * q[b][i][h] . K[b][g][k]) V[b][g][k]
 * over k in {0..ctx_b-1} and {ctx_b + j : mask bit (i, j)}; the caller has
 * written the N_b new tokens' keys and values at rows ctx_b..ctx_b+N_b-1.
 * Accumulation is fp32.  Rows i >= N_b of out are left untouched.
 *  d_q, d_out   [batch][n_max][hq][head_dim] (dtype)
 *  d_k, d_v     [batch][hkv][s_cap][head_dim] (dtype)
 *  max_ctx      host-side bound on every ctx_b (sizes the work split)
 *  d_workspace  ltd_attention_workspace_bytes() bytes of caller memory,
 *               zero-filled before its first use.  When the keys are split
 *               it holds per-split partial rows and per-unit counters; every
 *               call that ends without a device error leaves the counters
 *               at zero (after LTD_DEVERR_TIMEOUT, zero it again).  The size
 *               depends on the current device's SM count.
 * bf16 with head_dim 128 runs on the tcgen05 tensor cores; other shapes
 * (f32, head_dim in {32, 64, 96, 128}) run on a CUDA-core kernel. */
size_t ltd_attention_workspace_bytes(int32_t batch, int32_t hq, int32_t hkv, int32_t head_dim,
                                     int32_t n_max, int32_t max_ctx, ltd_dtype dtype);
ltd_status ltd_tree_attention(const void* d_q, const void* d_k, const void* d_v, void* d_out,
                              ltd_dtype dtype, int32_t batch, int32_t hq, int32_t hkv,
                              int32_t head_dim, int32_t s_cap, const int32_t* d_ctx,
                              int32_t max_ctx, const int32_t* d_n_verify, int32_t n_max,
                              const uint32_t* d_mask, float scale, void* d_workspace,
                              size_t workspace_bytes, ltd_stream_t stream);

/* ltd_tree_attention, and in addition a hint for the next call: once this
 * call has loaded its own keys and values, the tensor-core kernel asks L2 to
 * fetch the rows it just used from d_next_k / d_next_v (the next layer's
 * cache, same layout and sizes; the same ctx and N), so that the next call's
 * loads find them in L2 instead of HBM.  Results are identical to
 * ltd_tree_attention; the hint is skipped when one layer's keys and values
 * exceed 64 MB (they would crowd L2) and by the CUDA-core kernel.  The
 * paper has no counterpart: it is a deployment convenience for consecutive
 * layers.  d_next_k and d_next_v must both be valid 16-byte aligned device
 * pointers or both NULL (then this is ltd_tree_attention). */
ltd_status ltd_tree_attention_next(const void* d_q, const void* d_k, const void* d_v, void* d_out,
                                   ltd_dtype dtype, int32_t batch, int32_t hq, int32_t hkv,
                                   int32_t head_dim, int32_t s_cap, const int32_t* d_ctx,
                                   int32_t max_ctx, const int32_t* d_n_verify, int32_t n_max,
                                   const uint32_t* d_mask, float scale, void* d_workspace,
                                   size_t workspace_bytes, const void* d_next_k,
                                   const void* d_next_v, ltd_stream_t stream);

/* Which kernel ltd_tree_attention runs for these sizes: returns 1 for the
 * tcgen05 tensor-core kernel, 0 for the CUDA-core kernel, -1 if the sizes are
 * unsupported.  *launches (if not NULL) receives the number of kernel
 * launches one ltd_tree_attention call with these sizes makes. */
int32_t ltd_attention_kernel(ltd_dtype dtype, int32_t batch, int32_t hq, int32_t hkv,
                             int32_t head_dim, int32_t n_max, int32_t max_ctx, int32_t* launches);

/* KV cache views for compaction: device arrays of n_layers device pointers,
 * each layer [batch][hkv][s_cap][head_dim] of dtype. */
typedef struct ltd_kv_cache {
  void* const* d_k_layers;
  void* const* d_v_layers;
  int32_t n_layers, hkv, head_dim, s_cap;
  ltd_dtype dtype;
} ltd_kv_cache;

/* Acceptance (section 3.2 "Draft Tree Verification").
 * Greedy (d_mode[b] == LTD_GREEDY): from slot 0, repeatedly take the
 * target's argmax at the current slot (ties to the lower token id) and move
 * to the verified child carrying that token; stop at the first mismatch, the
 * argmax there is the bonus token.
 * Stochastic (LTD_STOCHASTIC, temperature 1; the paper only requires the
 * target distribution be preserved): at the current slot u, p = softmax of
 * the target row, q = softmax of the draft row that expanded u; each verified
 * child x_i in slot order is accepted if r_i q(x_i) < p(x_i), else
 * p <- max(p - q, 0) / sum; with no child accepted the bonus is the
 * Gumbel-max draw argmax_t log p(t) - log(-log g_t).  r_i and g_t are
 * counter-based uniforms: h = seed; h = mix64(h + 0x9E3779B97F4A7C15 (j+1)
 * + w_j) over the words (b, cycle, stream, slot, i-or-token), mix64 being the
 * splitmix64 finaliser; r = (h >> 40) 2^-24 (stream 0), g = (2 (h >> 41) + 1)
 * 2^-24 (stream 1).
 * Stochastic with point-mass proposals (LTD_STOCHASTIC_POINT_MASS, T = 1):
 * the children are deterministic top-k proposals, so each is treated as a
 * point mass on its token: child x_i is accepted if r_i (1 - p(R)) < p(x_i),
 * R the children rejected so far at this slot, else x_i joins R; with no
 * child accepted the bonus is the Gumbel-max draw over the tokens outside R.
 * The emitted token is distributed exactly as p for any set of children;
 * no draft row is read and a rejection costs no pass over the vocabulary.
 * Stochastic without replacement (LTD_STOCHASTIC_NO_REPLACEMENT, T = 1): as
 * LTD_STOCHASTIC, for children drawn from q without replacement: child x_i
 * is proposed by q_i = q with the rejected children removed, renormalised;
 * accept if r_i q_i(x_i) < p_i(x_i), else p_{i+1} = max(p_i - q_i, 0) / sum
 * and q_{i+1} = q_i without x_i, renormalised.
 *  d_target_logits  [batch][n_max][vocab] (dtype), row i = target at slot i
 *  d_draft_rows     the row store given to ltd_expand_tree (read by the
 *                   LTD_STOCHASTIC and LTD_STOCHASTIC_NO_REPLACEMENT rules)
 *  d_node_ids       ltd_select_verify output
 *  d_ctx            [batch] in; d_new_ctx [batch] out = ctx + 1 + accept_len
 *  d_path           out [batch][max_depth+1] accepted slots, -1 after the end
 *  d_accept_len     out [batch] accepted draft tokens (root excluded)
 *  d_bonus          out [batch]
 *  kv               if not NULL, the accepted rows are compacted in every
 *                   layer: row ctx+t <- row ctx+path[t] (ltd_kv_compact).
 *  d_workspace      ltd_accept_workspace_bytes() bytes of caller memory
 *                   (per-slot, per-vocabulary-chunk statistics); its contents
 *                   need no initial value and are overwritten by every call.
 * vocab above 262144 returns LTD_ERR_UNSUPPORTED: the stochastic walk keeps
 * p and q of one sequence in the shared memory of one 16-CTA cluster. */
size_t ltd_accept_workspace_bytes(int32_t batch, int32_t n_max, int64_t vocab);
ltd_status ltd_accept(const ltd_tree* tree, const void* d_target_logits,
                      const void* d_draft_rows, ltd_dtype dtype, int64_t vocab,
                      int64_t rows_per_seq, const int32_t* d_node_ids,
                      const int32_t* d_n_verify, int32_t n_max, const int32_t* d_mode,
                      uint64_t seed, uint64_t cycle, const int32_t* d_ctx, int32_t* d_new_ctx,
                      int32_t* d_path, int32_t* d_accept_len, int32_t* d_bonus,
                      const ltd_kv_cache* kv, void* d_workspace, size_t workspace_bytes,
                      ltd_stream_t stream);

/* ltd_accept at a sampling temperature T (section 5.1 "Metrics" reports
 * T = 1, where ltd_accept is this call with temperature 1): every stochastic
 * rule uses p = softmax(target row / T) and q = softmax(draft row / T) in
 * place of the plain softmaxes, the greedy rule is unchanged (the argmax does
 * not depend on T).  At T != 1 the walk reduces each visited draft row's
 * normaliser over its cluster (two more cluster barriers per node with
 * children); at T = 1 it uses the one the expansion stored, and the results
 * are bit for bit those of ltd_accept.
 *  temperature      > 0 and finite, else LTD_ERR_INVALID_ARG
 * Every other argument, the outputs and the errors as ltd_accept. */
ltd_status ltd_accept_tempered(const ltd_tree* tree, const void* d_target_logits,
                               const void* d_draft_rows, ltd_dtype dtype, int64_t vocab,
                               int64_t rows_per_seq, const int32_t* d_node_ids,
                               const int32_t* d_n_verify, int32_t n_max, const int32_t* d_mode,
                               float temperature, uint64_t seed, uint64_t cycle,
                               const int32_t* d_ctx, int32_t* d_new_ctx, int32_t* d_path,
                               int32_t* d_accept_len, int32_t* d_bonus, const ltd_kv_cache* kv,
                               void* d_workspace, size_t workspace_bytes, ltd_stream_t stream);

/* Acceptance for callers that cannot allocate device memory when they
 * accept a draft -- a serving loop that reserved its memory up front and
 * keeps allocation off the hot path, a plugin whose host framework owns all
 * device buffers, code that must stay allocation-free so its stream can be
 * captured with a fixed memory plan.  The paper has no counterpart; it is
 * a deployment convenience.
 *
 * Same arguments and results as ltd_accept without the workspace: the
 * scratch lives in a static device array of LTD_ACCEPT_NOALLOC_SCRATCH_BYTES
 * (1 MiB) inside the library, held by every GPU that loads it until the
 * process exits.  Sizes whose ltd_accept_workspace_bytes() exceeds that
 * return LTD_ERR_SHAPE.  Allocates nothing (no cudaMalloc or cudaFree) and
 * needs no part of the array cleared between calls.
 * The first call on a device looks up the array's device address; make
 * that first call before any stream capture.  All calls share the array,
 * so calls whose kernels overlap on the GPU (for example on two streams)
 * race; calls on one stream are ordered and safe. */
#define LTD_ACCEPT_NOALLOC_SCRATCH_BYTES (1u << 20)
ltd_status ltd_accept_noalloc(const ltd_tree* tree, const void* d_target_logits,
                              const void* d_draft_rows, ltd_dtype dtype, int64_t vocab,
                              int64_t rows_per_seq, const int32_t* d_node_ids,
                              const int32_t* d_n_verify, int32_t n_max, const int32_t* d_mode,
                              uint64_t seed, uint64_t cycle, const int32_t* d_ctx,
                              int32_t* d_new_ctx, int32_t* d_path, int32_t* d_accept_len,
                              int32_t* d_bonus, const ltd_kv_cache* kv, ltd_stream_t stream);

/* Write the verified tokens' new keys and values into every layer's cache,
 * at the rows tree attention reads them from (section 3.2, "Draft Tree
 * Verification": the target forward over the V candidates):
 *   cache_K[l][b][h][ctx_b + i] = d_new_k[l][b][h][i],  i < N_b,
 * and the same for V, in one launch for all layers.
 *  d_new_k, d_new_v  [n_layers][batch][hkv][n_max][head_dim] in the cache's
 *                    dtype (rows i >= N_b are not read)
 *  d_ctx, d_n_verify [batch]
 * A sequence with N_b outside [1, n_max] or ctx_b + N_b > s_cap is flagged
 * (LTD_DEVERR_NVERIFY / LTD_DEVERR_CTX) and its rows are left as they are.
 * Rows must be whole 16-byte units (LTD_ERR_UNSUPPORTED otherwise), the
 * arrays 16-byte aligned (LTD_ERR_INVALID_ARG otherwise). */
ltd_status ltd_kv_append(const ltd_kv_cache* kv, int32_t batch, int32_t n_max,
                         const void* d_new_k, const void* d_new_v, const int32_t* d_ctx,
                         const int32_t* d_n_verify, ltd_stream_t stream);

/* In-place KV compaction ("discards the remainder", section 3.2): for every
 * layer, sequence, KV head and K/V tensor, row ctx+t <- row ctx+path[t] for
 * t = 0..accept_len, every source read before any row is written.  Rows
 * below ctx and from ctx+accept_len+1 up are left as they are.
 *  d_path [batch][path_stride], d_accept_len [batch], d_ctx [batch] (the
 *  context before the cycle). */
ltd_status ltd_kv_compact(const ltd_kv_cache* kv, int32_t batch, const int32_t* d_path,
                          int32_t path_stride, const int32_t* d_accept_len,
                          const int32_t* d_ctx, ltd_stream_t stream);

/* The target's LM head over the verified tokens with the row statistics
 * acceptance reads (section 3.2, "Draft Tree Verification": one target
 * forward over the verified tokens; its last layer maps each hidden state
 * to vocabulary logits): logits[r][v] = sum_k hidden[r][k] weight[v][k]
 * (bf16 inputs, fp32 accumulation on the tensor cores) and per row the max,
 * the log-sum-exp and the argmax (ties to the lower token id), without the
 * logits making a round trip through memory.
 *  d_hidden        [rows][hidden] bf16, row-major, 16-byte aligned
 *  d_weight        [vocab][hidden] bf16, row-major, 16-byte aligned
 *  rows            1 .. LTD_LM_HEAD_MAX_ROWS (the verified tokens of a batch)
 *  hidden          a multiple of 64
 *  d_logits        [rows][vocab] bf16 out, or NULL to skip them (the
 *                  stochastic rules read full rows; greedy acceptance needs
 *                  only the argmax)
 *  d_row_max, d_row_lse  [rows] fp32 out; d_row_argmax [rows] int32 out
 *  d_workspace     ltd_lm_head_workspace_bytes() bytes of caller memory,
 *                  16-byte aligned; no initial value needed
 * Bad pointers are LTD_ERR_INVALID_ARG, bad sizes LTD_ERR_SHAPE
 * (ltd_lm_head_workspace_bytes returns 0 for them). */
#define LTD_LM_HEAD_MAX_ROWS 256
size_t ltd_lm_head_workspace_bytes(int32_t rows, int64_t vocab, int32_t hidden);
ltd_status ltd_lm_head_row_stats(const void* d_hidden, const void* d_weight, int32_t rows,
                                 int64_t vocab, int32_t hidden, void* d_logits, float* d_row_max,
                                 float* d_row_lse, int32_t* d_row_argmax, void* d_workspace,
                                 size_t workspace_bytes, ltd_stream_t stream);

/* Test hook of the bounded waits (section 3.2 has no counterpart; it exists
 * so the failure path can be exercised without a GPU fault).  With the keys
 * of each (sequence, KV head, tile) split over several CTAs, every split of
 * the tensor-core attention kernel waits on its unit's arrival counter for
 * the others; this sets, for the calls that follow on any thread, the
 * longest that wait lasts (limit_ns; 0 restores the default of one second)
 * and a number of arrivals it waits for beyond the unit's splits
 * (extra_arrivals; 0 restores normal operation).  Nothing ever supplies the
 * extra arrivals, so with extra_arrivals > 0 every split gives up after
 * limit_ns, raises LTD_DEVERR_TIMEOUT (ltd_check returns LTD_ERR_TIMEOUT),
 * leaves its rows of the output unwritten and still departs, so the
 * counters are back at zero and the workspace can be used again.
 * extra_arrivals above 1024 returns LTD_ERR_INVALID_ARG. */
ltd_status ltd_debug_attention_wait(uint64_t limit_ns, uint32_t extra_arrivals);

/* Test hook of the expansion's bounded wait (section 3.2 has no counterpart;
 * it exists so the failure path can be exercised without a GPU fault).  The
 * CTA that merges a sequence's rows in ltd_expand_tree waits until every
 * item record of the level carries the level's tag; this sets, for the
 * calls that follow on any thread, the longest that wait lasts (limit_ns; 0
 * restores the default of one second) and an offset added to the tag it
 * waits for (tag_offset; 0 restores normal operation).  No record ever
 * carries the offset tag, so with tag_offset > 0 every merging CTA gives
 * up after limit_ns, raises LTD_DEVERR_TIMEOUT (ltd_check returns
 * LTD_ERR_TIMEOUT) and leaves the level unbuilt: n_levels unchanged, so
 * the same level can be expanded again.  tag_offset above 1024 returns
 * LTD_ERR_INVALID_ARG. */
ltd_status ltd_debug_expand_wait(uint64_t limit_ns, uint32_t tag_offset);

/* Diagnostic of the tensor-core building blocks the attention kernel uses
 * (TMA with 128-byte swizzle, tcgen05.mma from shared-memory descriptors
 * into tensor memory, tcgen05.ld): one 128x128x128 bf16 GEMM with fp32
 * output.  mode 0: C = A B^T with B stored [N][K]; mode 1: C = A B with B
 * stored [K][N].  d_a, d_b row-major bf16 [128][128], d_c row-major fp32
 * [128][128], all 16-byte aligned device memory.  No counterpart in the
 * paper: it exists so a driver or toolkit change that breaks these
 * instructions shows up as a wrong product, not a wrong attention. */
ltd_status ltd_selftest_umma(int32_t mode, const void* d_a, const void* d_b, float* d_c,
                             ltd_stream_t stream);

/* Synchronise the stream, read and clear this device's error word.
 * Returns LTD_OK, LTD_ERR_TIMEOUT, LTD_ERR_DEVICE or LTD_ERR_CUDA; if
 * out_bits is not NULL it receives the raw LTD_DEVERR_* bits. */
ltd_status ltd_check(ltd_stream_t stream, uint32_t* out_bits);

/* Human-readable name of a status. */
const char* ltd_status_string(ltd_status status);

/* Version of this library as major*10000 + minor*100 + patch. */
int32_t ltd_version(void);

#ifdef __cplusplus
}
#endif

#endif /* LTD_H */
