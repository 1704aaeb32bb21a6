/*
 * adt.h - C ABI of libadt, the GPU tree-verify path of ADT-Tree
 * (Adjacency-Adaptive Dynamical Draft Trees, arXiv 2512.21857).
 *
 * One speculative-decoding step of a visual autoregressive model drafts a
 * tree of tokens, has the target model verify every node in one pass, keeps
 * the longest acceptable root path, and commits it to the KV cache (Sec. 3.1).
 * This library is the data-parallel part of that step, for one GPU:
 *
 *   adt_tree_expand   one layer of draft-tree growth: per frontier row, top-k
 *                     children and their path scores; the next frontier.
 *   adt_tree_rerank   the final tree: top-(N-1) candidates by score + root.
 *   adt_tree_attn     tree-masked attention of the N nodes over the prefix
 *                     KV cache and their own ancestors (one call per layer).
 *   adt_tree_accept   greedy / speculative-sampling walk: accepted path,
 *                     its length and the bonus token.
 *   adt_kv_compact    copy the accepted nodes' K/V into the cache.
 *   adt_ctrl_*        host-side depth / width controller (Sec. 4.1, 4.2).
 *
 * Conventions shared by every entry point
 *   - Pointers marked [device] are CUDA device pointers owned by the caller;
 *     the library never frees or retains them after the call returns.
 *   - GPU entry points are asynchronous and ordered on `stream` (a
 *     cudaStream_t passed as void*; NULL = the legacy default stream).  They
 *     launch kernels only: no allocation, no host synchronisation, so they
 *     can be captured in a CUDA graph.
 *   - Arguments are checked on the host before any launch; a violation
 *     returns ADT_ERR_INVALID_ARG (or ADT_ERR_UNSUPPORTED for valid but not
 *     implemented shapes) and launches nothing.
 *   - Conditions only the device can see (a malformed parent array, a KV
 *     length beyond the cache, an out-of-range path) set bits in a per-device
 *     error word and the offending work item is skipped; read and clear it
 *     with adt_get_device_error().
 *   - Workspace: a call that needs scratch memory takes (workspace,
 *     workspace_bytes); size it with the matching *_workspace_size() query.
 *     The workspace must be zero-filled once before its first use; every
 *     call leaves its completion counters (kept at fixed offsets at the
 *     start of the workspace) at zero again when it completes, so one
 *     workspace can serve any sequence of calls of the same entry point,
 *     of any shape, if it is as large as the largest query.  A workspace
 *     serves one entry point only, and calls that share it must not overlap
 *     in time.  After a call that reported a device error, zero it again.
 *   - bf16 tensors are raw IEEE bfloat16 bit patterns (adt_bf16).
 *   - Tree layout: B trees packed back to back.  node_offsets[b] ..
 *     node_offsets[b+1]-1 are the global indices of tree b's nodes; within a
 *     tree, node 0 is the root (the last committed token, whose K/V this
 *     pass produces) and parents[] holds tree-local indices with
 *     parents[0] = -1 and 0 <= parents[i] < i for i > 0.
 *   - No C++ exception crosses this boundary.
 */
#ifndef ADT_H_
#define ADT_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef uint16_t adt_bf16;

typedef enum adt_status {
  ADT_OK = 0,
  ADT_ERR_INVALID_ARG = 1,  /* rejected on the host, nothing launched       */
  ADT_ERR_UNSUPPORTED = 2,  /* valid request outside the implemented shapes */
  ADT_ERR_CUDA = 3,         /* a CUDA runtime call failed                   */
  ADT_ERR_TIMEOUT = 4,      /* a bounded device-side wait gave up           */
  ADT_ERR_WORKSPACE = 5,    /* workspace missing or too small               */
  ADT_ERR_DEVICE = 6        /* device error word was non-zero               */
} adt_status;

/* Bits of the device error word (adt_get_device_error). */
#define ADT_DEVERR_BAD_TREE 0x1u     /* parents[] violates the tree layout       */
#define ADT_DEVERR_KV_RANGE 0x2u     /* kv_len outside [0, max_kv] / cache room  */
#define ADT_DEVERR_BAD_PATH 0x4u     /* path / accept_len not a path of the tree */
#define ADT_DEVERR_TIMEOUT 0x8u      /* bounded wait expired                     */
#define ADT_DEVERR_BAD_INDEX 0x10u   /* candidate / token index out of range     */

typedef enum adt_accept_mode {
  /* T = 0: a child is accepted iff its token is the target argmax at the
   * parent (lowest index on ties); bonus = argmax at the last accepted node. */
  ADT_ACCEPT_GREEDY = 0,
  /* Eq. 1 per child, u * q(x) < p(x), with recursive rejection sampling
   * across siblings: after rejecting x, p <- max(0, p - q)/sum (unchanged if
   * that sum is 0) and q(x) <- 0, q <- q/sum.  Lossless when the children
   * were drawn without replacement from q. */
  ADT_ACCEPT_SPEC = 1,
  /* Deterministic candidates (q = 1 on the candidate, as for top-k drafts):
   * accept iff u < p(x); after a rejection p(x) <- 0 and p is renormalised.
   * Lossless for any fixed candidate set. */
  ADT_ACCEPT_SPEC_DET = 2
} adt_accept_mode;

/* Library version (major * 10000 + minor * 100 + patch). */
int32_t adt_version(void);

/* Reads the calling thread's current device's error word into *bits (may be
 * NULL), clears it, and synchronises `stream` first.  Returns ADT_OK when
 * the word was zero, ADT_ERR_DEVICE otherwise (ADT_ERR_CUDA on CUDA error). */
adt_status adt_get_device_error(void* stream, uint32_t* bits);

/* Human-readable name of a status code (static string). */
const char* adt_status_string(adt_status s);

/* Testing hook, not for production use.  Every wait of adt_tree_attn's
 * pipeline (a CTA waiting for its loads, products or softmax stages) is
 * bounded: after `polls` unsuccessful polls it gives up, sets
 * ADT_DEVERR_TIMEOUT in the device error word and the kernel leaves cleanly
 * (the copies and tensor-core products it already issued are waited for
 * first, so the device stays usable; the outputs of that call are
 * unspecified).  This sets the bound for the launches that follow in this
 * process; 0 restores the default (2^20 polls).  It lets a test make a
 * bounded wait run out without any fault; it is not synchronised with
 * calls on other threads. */
adt_status adt_testing_set_wait_limit(uint32_t polls);

/* Testing hook, not for production use: out[i] = e^(a[i] - b[i]) (a[i] <= b[i])
 * as the sampling modes of adt_tree_accept compute it, in double-float
 * arithmetic (two fp32 words; table-driven reduction), returned as fp64, so
 * that a test can bound its error against an fp64 exponential.  a, b
 * [device] fp32 [n]; out [device] fp64 [n]. */
adt_status adt_testing_exp_diff(const float* a, const float* b, int32_t n, double* out, void* stream);

/* ------------------------------------------------------------------------
 * adt_tree_attn - tree-masked attention for one transformer layer.
 *
 * Defines (Sec. 3.1: each draft node is verified conditioned on the prefix
 * and on its ancestor sequence ans(t) under the tree mask):
 *   for every tree b, node t of b, query head h (kv head g = h / (H/Hkv)):
 *     keys   = k_cache[b][g][0 .. kv_len[b]-1]  followed by  k_tree[j][g]
 *              for j in ans(t) and t itself (global indices of tree b)
 *     out[t][h] = softmax(softmax_scale * keys . q[t][h]) . values
 *     lse[t][h] = log sum exp(softmax_scale * keys . q[t][h])   (natural log)
 *
 * q       [device] bf16 [Ntot][H][D], row-major (Ntot = node_offsets[B]).
 * k_cache, v_cache [device] bf16; element (b, g, pos, d) at
 *         b*cache_stride_b + g*cache_stride_h + pos*D + d (strides in
 *         elements, multiples of 8).
 * kv_len  [device] int32 [B], prefix length of each tree, 0 <= kv_len <= max_kv.
 * k_tree, v_tree [device] bf16 [Ntot][Hkv][D].
 * parents [device] int32 [Ntot]; node_offsets [device] int32 [B+1].
 * B >= 1; H % Hkv == 0; D in {64, 128}; 1 <= max_nodes <= 256 with every
 *         tree no larger than max_nodes (larger trees are processed in
 *         query tiles of 64 nodes); max_kv >= every kv_len[b].
 * out     [device] bf16 [Ntot][H][D]; lse [device] fp32 [Ntot][H] or NULL.
 * All device pointers 16-byte aligned.  q/out must not alias the caches.
 * Nodes with a malformed tree set ADT_DEVERR_BAD_TREE and their rows are
 * left unspecified; kv_len[b] > max_kv sets ADT_DEVERR_KV_RANGE.
 * ------------------------------------------------------------------------ */
size_t adt_tree_attn_workspace_size(int32_t B, int32_t H, int32_t D, int32_t max_nodes,
                                    int32_t max_kv);

adt_status adt_tree_attn(const adt_bf16* q, const adt_bf16* k_cache, const adt_bf16* v_cache,
                         const int32_t* kv_len, int64_t cache_stride_b, int64_t cache_stride_h,
                         const adt_bf16* k_tree, const adt_bf16* v_tree, const int32_t* parents,
                         const int32_t* node_offsets, int32_t B, int32_t H, int32_t Hkv, int32_t D,
                         int32_t max_nodes, int32_t max_kv, float softmax_scale, adt_bf16* out,
                         float* lse, void* workspace, size_t workspace_bytes, void* stream);

/* ------------------------------------------------------------------------
 * adt_tree_attn_noalloc - adt_tree_attn without a workspace argument.
 *
 * The paper has no counterpart: this entry point exists for callers that
 * cannot allocate device memory themselves (a plugin whose host engine owns
 * every device allocation; a latency-critical thread that must not call
 * cudaMalloc, which may synchronise the device).  It computes what
 * adt_tree_attn computes, with the same arguments minus the workspace, and
 * allocates nothing: its scratch is one fixed 4 MiB array per device, held
 * by every GPU that loads the library until the process exits.
 *   - The first call on each device looks up that array's device address;
 *     make this first call before any stream capture begins.
 *   - Only launches whose key splits merge through memory use the array:
 *     more than 8 splits per (tree, query tile, head), which the split
 *     heuristic picks when B * ceil(max_nodes/64) * H is small.  They take
 *     B * ceil(max_nodes/64) * H * (4 + splits * 64 * (D + 2) * 4) bytes;
 *     where that exceeds 4 MiB the key range is cut into fewer splits (at
 *     most 8 of them merge on chip and need no scratch), so every shape
 *     this call accepts fits.  Shapes beyond the limits of adt_tree_attn
 *     (B * ceil(max_nodes/64) * H > 65536) return ADT_ERR_INVALID_ARG and
 *     launch nothing.
 *   - Every call shares the array, which keeps the last call's contents;
 *     the call clears what must start at zero (its completion counters) on
 *     `stream` itself.  Calls that overlap on the GPU (other streams, other
 *     host threads) race on it: serialise them.
 * ------------------------------------------------------------------------ */
adt_status adt_tree_attn_noalloc(const adt_bf16* q, const adt_bf16* k_cache,
                                 const adt_bf16* v_cache, const int32_t* kv_len,
                                 int64_t cache_stride_b, int64_t cache_stride_h,
                                 const adt_bf16* k_tree, const adt_bf16* v_tree,
                                 const int32_t* parents, const int32_t* node_offsets, int32_t B,
                                 int32_t H, int32_t Hkv, int32_t D, int32_t max_nodes,
                                 int32_t max_kv, float softmax_scale, adt_bf16* out, float* lse,
                                 void* stream);

/* ------------------------------------------------------------------------
 * adt_tree_expand - one layer of dynamic draft-tree growth (Sec. 3.1 last
 * paragraph; Sec. 4.2 / Fig. 5; node score Eq. 4 in the log domain).
 *
 * For each frontier row r < F, x = logits[r] / temperature (fp32):
 *   the k_child largest entries (value desc, lowest index on ties; -0 == +0)
 *   become children r*k_child + j, j = 0 .. k_child-1, with
 *     child_logp  = x_tok - log sum_v exp(x_v)        (log q(tok), fp32)
 *     child_score = frontier_score[r] + child_logp     (log path confidence)
 *     child_parent = frontier_id[r] (or r if frontier_id is NULL)
 * keep_idx = the k_keep candidates with the highest child_score (lowest
 * candidate index on ties), best first; next_score / next_id are their
 * scores and child_id_base + keep_idx, i.e. the next call's frontier.
 *
 * logits  [device] fp32, row r at logits + r*ld (ld >= V, multiple of 4).
 * frontier_score [device] fp32 [F]; frontier_id [device] int32 [F] or NULL.
 * 1 <= F <= 4096; 1 <= V <= 2^24; 1 <= k_child <= min(V, 64);
 * 1 <= k_keep <= min(F*k_child, 1024); temperature > 0.
 * child_token, child_parent [device] int32 [F*k_child];
 * child_logp (or NULL), child_score [device] fp32 [F*k_child];
 * keep_idx [device] int32 [k_keep]; next_score, next_id [device] or NULL.
 * keep_idx may be NULL (then next_score and next_id must be NULL too) when
 * no next frontier is wanted, e.g. for the tree's last layer: the children
 * are written as above and the selection across rows is skipped.
 * Logits must be finite (NaN is outside the domain and not checked).
 * ------------------------------------------------------------------------ */
size_t adt_tree_expand_workspace_size(int32_t F, int32_t V, int32_t k_child);

adt_status adt_tree_expand(const float* logits, int64_t ld, const float* frontier_score,
                           const int32_t* frontier_id, int32_t F, int32_t V, int32_t k_child,
                           int32_t k_keep, float temperature, int32_t child_id_base,
                           int32_t* child_token, float* child_logp, float* child_score,
                           int32_t* child_parent, int32_t* keep_idx, float* next_score,
                           int32_t* next_id, void* workspace, size_t workspace_bytes,
                           void* stream);

/* ------------------------------------------------------------------------
 * adt_tree_expand_cfg - adt_tree_expand on classifier-free-guided logits.
 * The paper computes the draft distribution q under classifier-free guidance
 * (Sec. 3.1, the sentence under Eq. 1; Fig. 5's conditional and
 * unconditional draft branches) with guidance scale 3.0 (Sec. 5.1).  Row r's
 * logits are formed on the fly from the two branches,
 *     l = uncond + cfg_scale * (cond - uncond),
 * each operation rounded to fp32 as written, then divided by temperature;
 * everything else is adt_tree_expand.
 *
 * logits_cond, logits_uncond [device] fp32, row r at + r*ld, same ld, both
 *         16-byte aligned; cfg_scale finite.  Other arguments and the
 *         workspace as for adt_tree_expand (one workspace serves both).
 * ------------------------------------------------------------------------ */
adt_status adt_tree_expand_cfg(const float* logits_cond, const float* logits_uncond, int64_t ld,
                               float cfg_scale, const float* frontier_score, const int32_t* frontier_id,
                               int32_t F, int32_t V, int32_t k_child, int32_t k_keep, float temperature,
                               int32_t child_id_base, int32_t* child_token, float* child_logp,
                               float* child_score, int32_t* child_parent, int32_t* keep_idx,
                               float* next_score, int32_t* next_id, void* workspace,
                               size_t workspace_bytes, void* stream);

/* ------------------------------------------------------------------------
 * adt_tree_rerank - the final draft tree (Eq. 4 and the sentence after it:
 * the top-N nodes by score form the tree that the target verifies).
 *
 * Candidates c < C are numbered depth-major (what successive expand calls
 * with child_id_base = running count produce); cand_parent[c] is the
 * parent's candidate index or -1 for a child of the root.  The n_nodes-1
 * candidates with the highest score (lowest index on ties) are emitted in
 * ascending candidate index as nodes 1 .. n_nodes-1 after the root (node 0,
 * token *root_token):
 *   tokens[i], parents[i] (tree-local), cand_index[i] (-1 for the root),
 *   depth[i] (0 for the root).
 * A chosen candidate whose parent was not chosen sets ADT_DEVERR_BAD_TREE.
 *
 * cand_token [device] int32 [C]; cand_score [device] fp32 [C];
 * cand_parent [device] int32 [C]; root_token [device] int32 [1].
 * 1 <= n_nodes <= C + 1; C <= 65536; n_nodes <= 4096.
 * tokens, parents [device] int32 [n_nodes]; cand_index, depth: same or NULL.
 * ------------------------------------------------------------------------ */
size_t adt_tree_rerank_workspace_size(int32_t C);

adt_status adt_tree_rerank(const int32_t* cand_token, const float* cand_score,
                           const int32_t* cand_parent, int32_t C, const int32_t* root_token,
                           int32_t n_nodes, int32_t* tokens, int32_t* parents,
                           int32_t* cand_index, int32_t* depth, void* workspace,
                           size_t workspace_bytes, void* stream);

/* ------------------------------------------------------------------------
 * adt_tree_accept - verification walk of each tree (Sec. 3.1, Eq. 1).
 *
 * Starting at the root, the children of the current node v are tried in
 * ascending node index under `mode` (see adt_accept_mode); p and q are
 * softmax(row / temperature) of v's target and draft rows.  An accepted
 * child becomes v; otherwise (or at a leaf) the walk stops and the bonus
 * token is drawn from the current p by inverse CDF: the smallest index t
 * with sum_{j<=t} p_j > u_sample[v] * sum_j p_j (GREEDY: argmax).
 *
 * target_logits [device] fp32, row of global node n at target + n*ld_target.
 * draft_logits  [device] fp32 (SPEC only, else may be NULL); the draft row
 *         of node n is draft + draft_row[n]*ld_draft, or + n*ld_draft when
 *         draft_row is NULL.  Only nodes with children have their draft row
 *         read: a leaf may map to -1.  A node with children and a negative
 *         draft_row sets ADT_DEVERR_BAD_INDEX and the walk stops there, its
 *         bonus drawn from the target distribution; non-negative rows are
 *         not range-checked (each must be a row of draft_logits).
 * tokens, parents [device] int32 [Ntot]; node_offsets [device] int32 [B+1].
 * u_accept, u_sample [device] fp32 [Ntot] in [0, 1) (SPEC modes; GREEDY may
 *         pass NULL): u_accept[n] decides child n, u_sample[v] draws the
 *         bonus at v.
 * 1 <= B; 1 <= V <= 262144; max_nodes >= every tree size; ld >= V, ld % 4 == 0.
 * path [device] int32 [B][max_path]: tree-local nodes of the accepted path,
 *         root first, padded with -1 (a path longer than max_path is cut and
 *         sets ADT_DEVERR_BAD_PATH).
 * accept_len [device] int32 [B] (= accepted draft nodes, path length - 1).
 * bonus_token [device] int32 [B].
 * ------------------------------------------------------------------------ */
size_t adt_tree_accept_workspace_size(int32_t B, int32_t V);

adt_status adt_tree_accept(const float* target_logits, int64_t ld_target,
                           const float* draft_logits, int64_t ld_draft, const int32_t* draft_row,
                           const int32_t* tokens, const int32_t* parents,
                           const int32_t* node_offsets, int32_t B, int32_t V, int32_t max_nodes,
                           const float* u_accept, const float* u_sample, adt_accept_mode mode,
                           float temperature, int32_t* path, int32_t max_path,
                           int32_t* accept_len, int32_t* bonus_token, void* workspace,
                           size_t workspace_bytes, void* stream);

/* ------------------------------------------------------------------------
 * adt_tree_accept_cfg - adt_tree_accept with p and q computed under
 * classifier-free guidance (Sec. 3.1, the sentence under Eq. 1; guidance
 * scale 3.0 in Sec. 5.1).  Every target (and, in SPEC mode, draft) row is
 * formed on the fly as uncond + cfg_scale * (cond - uncond), each operation
 * rounded to fp32 as written, before the division by temperature; the walk
 * is that of adt_tree_accept.
 *
 * target_cond, target_uncond [device] fp32, same layout and ld_target.
 * draft_cond, draft_uncond   [device] fp32, same layout and ld_draft (SPEC
 *         mode only, else may be NULL); draft_row maps nodes to rows as in
 *         adt_tree_accept.  cfg_scale finite.  Other arguments as for
 *         adt_tree_accept.
 * ------------------------------------------------------------------------ */
adt_status adt_tree_accept_cfg(const float* target_cond, const float* target_uncond, int64_t ld_target,
                               const float* draft_cond, const float* draft_uncond, int64_t ld_draft,
                               const int32_t* draft_row, float cfg_scale, const int32_t* tokens,
                               const int32_t* parents, const int32_t* node_offsets, int32_t B, int32_t V,
                               int32_t max_nodes, const float* u_accept, const float* u_sample,
                               adt_accept_mode mode, float temperature, int32_t* path, int32_t max_path,
                               int32_t* accept_len, int32_t* bonus_token, void* workspace,
                               size_t workspace_bytes, void* stream);

/* ------------------------------------------------------------------------
 * adt_kv_compact - commit the accepted path to the KV cache, all layers in
 * one launch (accepted tokens extend the prefix s_{1:t}, Sec. 3.1).
 *
 * For every layer l < num_layers, tree b and i = 0 .. accept_len[b]
 * (the root included):
 *   cache[l][b][g][kv_len[b] + i][:] <- tree[l][node_offsets[b] + path[b][i]][g][:]
 * for K and V and every kv head g.  kv_len_out[b] = kv_len[b] + accept_len[b] + 1.
 *
 * k_cache, v_cache [device] bf16; element (l, b, g, pos, d) at
 *         l*cache_layer_stride + b*cache_stride_b + g*cache_stride_h + pos*D + d.
 * k_tree, v_tree [device] bf16; element (l, n, g, d) at
 *         l*tree_layer_stride + n*Hkv*D + g*D + d.
 * kv_len [device] int32 [B]; kv_len_out [device] int32 [B] or NULL (must not
 *         alias kv_len).  path [device] int32 [B][max_path];
 * accept_len [device] int32 [B]; node_offsets [device] int32 [B+1].
 * D in {64, 128}; strides multiples of 8 elements; pointers 16-byte aligned.
 * kv_len[b] + accept_len[b] + 1 > max_kv (the cache capacity) or a path
 * entry outside the tree sets a device error bit and skips tree b.
 * The tree buffers must not overlap the cache.
 * ------------------------------------------------------------------------ */
adt_status adt_kv_compact(adt_bf16* k_cache, adt_bf16* v_cache, const int32_t* kv_len,
                          int32_t* kv_len_out, const adt_bf16* k_tree, const adt_bf16* v_tree,
                          const int32_t* node_offsets, const int32_t* path, int32_t max_path,
                          const int32_t* accept_len, int32_t B, int32_t Hkv, int32_t D,
                          int32_t num_layers, int32_t max_kv, int64_t cache_layer_stride,
                          int64_t cache_stride_b, int64_t cache_stride_h,
                          int64_t tree_layer_stride, void* stream);

/* ------------------------------------------------------------------------
 * adt_kv_compact_inplace - adt_kv_compact for a cache that already holds
 * the tree's K/V in its tail (the tree written right after the prefix, as
 * engines that append draft tokens to the cache do): row kv_len[b] + t of
 * tree b holds node t (local index).  For every layer l, tree b, kv head g
 * and i = 0 .. accept_len[b]:
 *   cache'[l][b][g][kv_len[b] + i][:] = cache[l][b][g][kv_len[b] + path[b][i]][:]
 * computed from the cache as it was before the call (a destination row may
 * be the source of another path entry; the kernel reads every moved row
 * before it writes any).  kv_len_out[b] = kv_len[b] + accept_len[b] + 1.
 * Rows of the tree past the new length are left as they were.
 *
 * Arguments as for adt_kv_compact, without the tree buffers;
 * node_offsets[b+1] - node_offsets[b] is tree b's size n_b, and
 * kv_len[b] + n_b <= max_kv.  1 <= max_path <= 256 (ADT_ERR_UNSUPPORTED
 * above).  A path entry outside the tree, or a tree that does not fit,
 * sets a device error bit and skips tree b.
 * ------------------------------------------------------------------------ */
adt_status adt_kv_compact_inplace(adt_bf16* k_cache, adt_bf16* v_cache, const int32_t* kv_len,
                                  int32_t* kv_len_out, const int32_t* node_offsets,
                                  const int32_t* path, int32_t max_path, const int32_t* accept_len,
                                  int32_t B, int32_t Hkv, int32_t D, int32_t num_layers,
                                  int32_t max_kv, int64_t cache_layer_stride,
                                  int64_t cache_stride_b, int64_t cache_stride_h, void* stream);

/* ------------------------------------------------------------------------
 * Depth / width controller (host only, no GPU).  Sec. 4.1 adjacent
 * initialisation, Eq. 2 bisectional adaptation, bounds at the end of
 * Sec. 4.2, hyper-parameters Sec. 5.1.  For the tree that emits grid
 * position pos = (i, j) (raster order, W = grid_w):
 *   init  horizontal: (d, k) of the tree that emitted pos-1 (the left
 *         neighbour; its raster predecessor across a row end);
 *         vertical: of the tree that emitted pos-W, horizontal if i = 0 or
 *         not generated; random: d ~ U{d_lo..d_hi}, k ~ U{k_lo..k_hi} from
 *         SplitMix64(seed + c*0x9E3779B97F4A7C15), c = 2*pos (d), 2*pos+1 (k);
 *         tokenflock (the Table 3 alternative): the weighted mean over the
 *         generated positions q < pos within distance delta = flock_delta,
 *         (x_q - x)^2 + (y_q - y)^2 <= delta^2 (x column, y row), with
 *         weights delta + 1 - (y - y_q) (the paper's (delta - dy + 1)/delta,
 *         normalised), rounded half up;
 *         (d0, k0) when nothing precedes; fix_d / fix_k > 0 override.
 *   adapt alpha = a / d of the previous tree: alpha >= beta -> (d+l_d, k-l_k),
 *         else (d-l_d, k+l_k); no adaptation for an image's first tree.
 *   clamp d to [d_lo, d_hi]; k to [k_lo, k_hi] when clamp_k_always or the
 *         adapted depth exceeds 1, else to [1, k_cap].
 * The paper's open bounds (0,10) / (3,14) are the closed [1,9] / [4,13].
 * ------------------------------------------------------------------------ */
enum { ADT_INIT_HORIZONTAL = 0, ADT_INIT_VERTICAL = 1, ADT_INIT_RANDOM = 2, ADT_INIT_TOKENFLOCK = 3 };

typedef struct adt_ctrl_params {
  double beta;
  int32_t l_d, l_k;
  int32_t d_lo, d_hi, k_lo, k_hi;
  int32_t init_mode;
  int32_t d0, k0;
  int32_t clamp_k_always;
  int32_t k_cap;
  int32_t fix_d, fix_k;
  uint64_t seed;
  int32_t flock_delta; /* tokenflock neighbourhood radius, >= 1 */
} adt_ctrl_params;

typedef struct adt_ctrl adt_ctrl; /* opaque; one per image */

/* Creates a controller for a grid_h x grid_w token grid.  Checks
 * 1 <= d_lo <= d_hi, 1 <= k_lo <= k_hi <= k_cap, l_d, l_k >= 0, d0, k0 >= 1,
 * 1 <= flock_delta <= 64 for tokenflock, grid sizes >= 1.  *out receives a heap object freed by adt_ctrl_destroy. */
adt_status adt_ctrl_create(const adt_ctrl_params* params, int32_t grid_h, int32_t grid_w,
                           adt_ctrl** out);
void adt_ctrl_destroy(adt_ctrl* ctrl);
/* (d, k) for the tree that will emit position pos (0 <= pos < grid_h*grid_w). */
adt_status adt_ctrl_next(adt_ctrl* ctrl, int32_t pos, int32_t* depth, int32_t* width);
/* Records the verify result of the tree from the latest adt_ctrl_next:
 * 0 <= accept_len <= depth; positions pos .. pos+accept_len remember (d, k);
 * *next_pos (may be NULL) = pos + accept_len + 1. */
adt_status adt_ctrl_update(adt_ctrl* ctrl, int32_t pos, int32_t accept_len, int32_t* next_pos);
/* Checkpoint / resume: the controller's whole state (parameters, grids,
 * the previous tree's acceptance rate) as bytes.  adt_ctrl_state_size gives
 * the size (0 for NULL); adt_ctrl_save writes it into buf (bytes >= size);
 * adt_ctrl_load creates a controller from saved bytes (freed by
 * adt_ctrl_destroy), rejecting buffers that are short or not a saved
 * state.  Host byte order: a checkpoint for the same build. */
size_t adt_ctrl_state_size(const adt_ctrl* ctrl);
adt_status adt_ctrl_save(const adt_ctrl* ctrl, void* buf, size_t bytes);
adt_status adt_ctrl_load(const void* buf, size_t bytes, adt_ctrl** out);
/* The (d, k) recorded for a generated position (0, 0 if not generated). */
adt_status adt_ctrl_get(const adt_ctrl* ctrl, int32_t pos, int32_t* depth, int32_t* width);

#ifdef __cplusplus
}
#endif

#endif /* ADT_H_ */
