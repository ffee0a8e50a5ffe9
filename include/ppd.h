/*
 * ppd.h -- C ABI of libppd, the GB300 (sm_103a) implementation of the
 * verification step of Parallel Prompt Decoding (PPD).
 *
 * One PPD decode step runs a single forward pass over a token tree: the root
 * (the last accepted token), candidate ("guess") tokens, and a chain of prompt
 * tokens hanging below each candidate (paper Section 3; Section 4.1).  The
 * verification part of that step, which this library implements, is:
 *
 *   1. tree-masked attention: every tree token attends to the KV-cache prefix,
 *      its tree ancestors and itself (Section 3, step (1), tree attention;
 *      Section 4.1, the tree attention mask);
 *   2. node argmax: the model's top-1 token after every tree node (the greedy
 *      exact-matching check of Section 3, step (2));
 *   3. acceptance: the longest root-to-node path whose every candidate equals
 *      the top-1 token at its parent (Section 3, steps (2)-(3));
 *   4. compaction: the accepted nodes' K/V rows enter the cache (Section 3,
 *      step (3): the accepted rows are appended to the cache).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - All tensor pointers are DEVICE memory, row-major (last index fastest),
 *    owned by the caller.  The library never allocates, frees or synchronises;
 *    work is enqueued on `stream` (a cudaStream_t passed as void*; NULL = the
 *    legacy default stream).  A PPD_OK return means the arguments passed the
 *    host-side checks and the work was enqueued; errors found on the device
 *    are reported per sequence in `dev_status`.
 *  - Shapes: L layers, B sequences, H heads (K/V heads == query heads), D head
 *    dim (64 or 128), T tree tokens (1..512), S_max cache rows per
 *    (layer, sequence, head), V vocab size.
 *  - Q, tree K/V and the attention output are [L,B,H,T,D]; the K/V cache is
 *    [L,B,H,S_max,D]; rows [0, prefix_len[b]) of sequence b are the valid
 *    prefix.  Q/K/V are bf16 (PPD_BF16) or fp32 (PPD_F32, rounded to bf16 on
 *    load, round-to-nearest-even).  Attention accumulates in fp32.
 *  - parent[b][0] = -1 and 0 <= parent[b][i] < i (topological order).  Trees
 *    may differ per sequence.  cand_tokens[b][i] is the token id of node i:
 *    in [0, V) for the root and the candidates, -1 for prompt-token nodes.
 *  - Argmax ties break to the lowest index; NaN ranks above every number and
 *    the first NaN wins; -0 equals +0.
 *  - The default softmax scale (scale <= 0) is 1/sqrt(D).
 *  - Tree buffers must not overlap the cache buffers.
 *
 * Per-sequence device status (dev_status[b]): PPD_OK, PPD_ERR_TREE (malformed
 * parent array, or a token id out of range), PPD_ERR_CAPACITY (prefix_len
 * outside [0, S_max], or prefix_len + accepted length > S_max), or
 * PPD_ERR_TIMEOUT (an internal wait gave up; the outputs of that call are
 * undefined).  A sequence with a non-zero status gets accept_len 0, path all
 * -1, next_token -1, new_prefix_len = prefix_len, and no cache write.
 */
#ifndef PPD_H
#define PPD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    PPD_OK = 0,
    PPD_ERR_INVALID_ARG = 1, /* host-side argument check failed; nothing enqueued */
    PPD_ERR_UNSUPPORTED = 2, /* valid request outside what this build supports */
    PPD_ERR_TREE = 3,        /* device: malformed tree or token id */
    PPD_ERR_CAPACITY = 4,    /* device: prefix / accepted rows exceed S_max */
    PPD_ERR_CUDA = 5,        /* a CUDA runtime call failed */
    PPD_ERR_TIMEOUT = 6      /* device: a bounded internal wait expired */
} ppd_status;

typedef enum { PPD_BF16 = 0, PPD_F32 = 1 } ppd_dtype;

/*
 * Scratch bytes the entry points below need in `workspace` for these sizes
 * (device memory, any contents, 256-byte aligned, caller-owned; it may be
 * reused between calls that are ordered on one stream).  Covers the per-split
 * partial maxima (and softmax statistics) of the node argmax, the fused step's
 * per-CTA scratch, for PPD_F32 the bf16 copies of Q/K/V, and the attention
 * work split's per-SM records and partial softmax states.
 */
size_t ppd_workspace_bytes(int L, int B, int H, int T, int D, int V, int S_max, ppd_dtype dt);

/*
 * Tree-masked attention (Section 3 step (1), Section 4.1).  For every layer l,
 * sequence b, head h and tree node i:
 *     o = sum_j softmax_j(scale * <q_i, k_j>) v_j
 * over the keys j in {cache rows 0..prefix_len[b]-1} U {tree nodes on the
 * path from i to the root, i included}.
 *   q, k_tree, v_tree  [L,B,H,T,D]      k_cache, v_cache [L,B,H,S_max,D]
 *   prefix_len int32[B]                 parent int32[B,T]
 *   out  fp32 [L,B,H,T,D]               lse  fp32 [L,B,H,T] natural-log
 *                                       log-sum-exp of the scaled scores, or NULL
 *   dev_status int32[B] (required): set to 0, or to PPD_ERR_TREE /
 *   PPD_ERR_CAPACITY / PPD_ERR_TIMEOUT; outputs of a failed sequence are
 *   unspecified.  Cache rows at or beyond prefix_len[b] are never used and may
 *   hold anything, NaN included.
 * Workspace: ppd_workspace_bytes(...) bytes.  With it (and B <= 64) the
 * (layer, sequence, head) slices left over after full rounds of one slice per
 * SM -- all of them, when there are fewer slices than SMs -- are shared out
 * over every SM by their key tiles, the slices cut between SMs being merged by
 * a second, small grid; a bf16 call may pass none (NULL or fewer bytes) and
 * then runs one whole slice per SM at a time.
 */
ppd_status ppd_tree_attention(const void *q, const void *k_cache, const void *v_cache,
                              const void *k_tree, const void *v_tree,
                              const int32_t *prefix_len, const int32_t *parent,
                              int L, int B, int H, int T, int D, int S_max, ppd_dtype dt,
                              float scale, float *out, float *lse, int32_t *dev_status,
                              void *workspace, size_t ws_bytes, void *stream);

/*
 * Node argmax (Section 3 step (2), exact matching needs the top-1 token after
 * every tree node).  logits fp32 [B,T,V] -> argmax_out int32 [B,T], lowest
 * index on ties, first NaN wins.  Workspace: ppd_workspace_bytes(...) bytes.
 */
ppd_status ppd_node_argmax(const float *logits, int B, int T, int V, int32_t *argmax_out,
                           void *workspace, size_t ws_bytes, void *stream);

/*
 * Exact-matching acceptance (Section 3 steps (2)-(3)).  Node 0 is always
 * accepted; node i > 0 is accepted when cand_tokens[b][i] >= 0 equals
 * argmax[b][parent[b][i]] and its parent is accepted.  The end node is the
 * deepest accepted node (smallest index among equal depths).
 *   argmax, cand_tokens, parent int32[B,T]; prefix_len int32[B]
 *   accept_len int32[B]   accepted tokens, root included (>= 1 on success)
 *   path int32[B,T]       accepted node ids in depth order, then -1
 *   next_token int32[B]   argmax at the end node (the next root token)
 *   new_prefix_len int32[B] = prefix_len + accept_len
 *   dev_status int32[B]   see the file header
 */
ppd_status ppd_accept_path(const int32_t *argmax, const int32_t *cand_tokens,
                           const int32_t *parent, const int32_t *prefix_len,
                           int B, int T, int V, int S_max,
                           int32_t *accept_len, int32_t *path, int32_t *next_token,
                           int32_t *new_prefix_len, int32_t *dev_status, void *stream);

/*
 * KV compaction (Section 3 step (3)).  For every l, b, h and j <
 * accept_len[b]:  cache[l,b,h,prefix_len[b]+j,:] <- tree[l,b,h,path[b][j],:]
 * for K and V, bit for bit (2 bytes per element for PPD_BF16, 4 for PPD_F32).
 * No other cache row is written.  Rows whose source or destination index is
 * out of range are skipped.
 */
ppd_status ppd_kv_compact(void *k_cache, void *v_cache, const void *k_tree, const void *v_tree,
                          const int32_t *path, const int32_t *accept_len,
                          const int32_t *prefix_len, int L, int B, int H, int T, int D,
                          int S_max, ppd_dtype dt, void *stream);

/*
 * The whole verification step (Section 3 steps (1)-(3)): node argmax and
 * acceptance, tree-masked attention over all L layers, and compaction of the
 * accepted rows, enqueued on `stream` with no host synchronisation.  For
 * B <= 64 the attention grid does the other steps with one spare warp per CTA
 * while its other warps stream K/V: that warp combines the argmax, decides
 * acceptance and compacts.  When the logits are at most 1/64 of the K/V bytes
 * (counted over S_max + T rows), those warps also compute the argmax partial
 * maxima themselves and the step is a single cooperative grid (the CTAs
 * exchange flags in the workspace, tagged with a per-call epoch that the
 * workspace also holds, so its contents still do not matter); otherwise an
 * argmax grid runs first and the attention grid may start while it runs.
 * If the cooperative launch cannot have every CTA resident, the step falls
 * back to the two-grid form.  Larger batches run the steps as separate grids.
 * Arguments as in the four entry points above; `out`/`lse` as in
 * ppd_tree_attention, `argmax_out` as in ppd_node_argmax.  Attention reads
 * only prefix rows [0, prefix_len[b]) and compaction writes only rows
 * [prefix_len[b], new_prefix_len[b]), so the result equals running the four
 * steps one after another.  The epoch word and the flags sit in the first
 * 2,064 bytes of the workspace at the same place for every size, so a
 * workspace may be reused across sizes (a flag only ever holds the tag of an
 * earlier call, below the next call's).  After a call that reported
 * PPD_ERR_TIMEOUT, fill the workspace with zeros before reusing it.
 */
ppd_status ppd_verify_step(const void *q, void *k_cache, void *v_cache,
                           const void *k_tree, const void *v_tree,
                           const int32_t *prefix_len, const int32_t *parent,
                           const int32_t *cand_tokens, const float *logits,
                           int L, int B, int H, int T, int D, int V, int S_max, ppd_dtype dt,
                           float scale, float *out, float *lse, int32_t *argmax_out,
                           int32_t *accept_len, int32_t *path, int32_t *next_token,
                           int32_t *new_prefix_len, int32_t *dev_status,
                           void *workspace, size_t ws_bytes, void *stream);

/*
 * Node softmax statistics for typical acceptance (Section 3 step (2): the
 * paper's second verification scheme, typical acceptance, tests each candidate
 * against the distribution predicted at its parent).  For every row of logits
 * fp32 [B,T,V], with p = softmax(logits / temperature):
 *   argmax_out  int32 [B,T]  top-1 index (lowest index on ties, first NaN wins)
 *   lse_out     fp32 [B,T]   log sum_v exp(logits_v / temperature)
 *   entropy_out fp32 [B,T]   -sum_v p_v log p_v (natural log)
 * A row holding a NaN gives NaN statistics.  temperature > 0.  One pass over the
 * logits.  Workspace: ppd_workspace_bytes(...) bytes.
 */
ppd_status ppd_node_stats(const float *logits, int B, int T, int V, float temperature,
                          int32_t *argmax_out, float *lse_out, float *entropy_out,
                          void *workspace, size_t ws_bytes, void *stream);

/*
 * Typical acceptance (Section 3 steps (2)-(3); the paper names the scheme and
 * gives no formula, so the rule below is the one this library adopts).  Node 0
 * is always accepted; node i > 0 with parent j and candidate token
 * t = cand_tokens[b][i] >= 0 is accepted when its parent is accepted and
 *     p_t > min(epsilon, delta * exp(-H_j)),
 * where p = softmax(logits[b][j] / temperature) and H_j its entropy, taken from
 * lse / entropy (as written by ppd_node_stats at the same temperature).  Path
 * choice (deepest accepted node, smallest index among equal depths), outputs and
 * errors as in ppd_accept_path; next_token is the argmax at the end node.
 *   logits fp32 [B,T,V]; lse, entropy fp32 [B,T]; argmax, cand_tokens, parent
 *   int32 [B,T]; prefix_len int32 [B].  temperature > 0; epsilon, delta finite.
 * A decision whose two sides agree to within float rounding may differ from a
 * higher-precision evaluation.
 */
ppd_status ppd_typical_accept(const float *logits, const float *lse, const float *entropy,
                              const int32_t *argmax, const int32_t *cand_tokens,
                              const int32_t *parent, const int32_t *prefix_len, int B, int T,
                              int V, int S_max, float temperature, float epsilon, float delta,
                              int32_t *accept_len, int32_t *path, int32_t *next_token,
                              int32_t *new_prefix_len, int32_t *dev_status, void *stream);

/*
 * The verification step with typical acceptance in place of exact matching:
 * ppd_verify_step's arguments plus temperature, epsilon and delta of
 * ppd_typical_accept.  argmax_out still receives every node's top-1 token.
 */
ppd_status ppd_verify_step_typical(const void *q, void *k_cache, void *v_cache,
                                   const void *k_tree, const void *v_tree,
                                   const int32_t *prefix_len, const int32_t *parent,
                                   const int32_t *cand_tokens, const float *logits,
                                   int L, int B, int H, int T, int D, int V, int S_max,
                                   ppd_dtype dt, float scale, float temperature, float epsilon,
                                   float delta, float *out, float *lse, int32_t *argmax_out,
                                   int32_t *accept_len, int32_t *path, int32_t *next_token,
                                   int32_t *new_prefix_len, int32_t *dev_status,
                                   void *workspace, size_t ws_bytes, void *stream);

/*
 * Next-step candidate tree (Section 3 step (1): the prompt tokens appended to a
 * guess token predict the tokens after it; Section 3, Ensemble Prompt Tokens:
 * each prompt position holds n_ept tokens, the j-th attending only to the j-th
 * of the earlier positions, and the guess comes from the average of their
 * logits; Appendix, Definition of tree states: the tree takes state T_k, whose
 * candidate subtree is at most k deep, k being the number of prompt positions
 * available below the accepted token).
 *   e = path[b][accept_len[b]-1], the accepted end node of sequence b.  The
 *   first n_ept children of e with cand_tokens -1 (index order) head n_ept
 *   prompt chains, each continued by the lowest-index such child of its last
 *   node; k = the shortest chain's length (0 when e has fewer than n_ept
 *   prompt children), capped at n_states - 1.  The guesses for depth d are
 *   the K best tokens (ranking: NaN first, then larger value, then lower index)
 *   of the fp32 average of the chains' logits at position d: summed in chain
 *   order, then divided by n_ept with IEEE rounding.  n_ept = 1: one chain,
 *   plain logits.  ppd_next_tree_ept with ept_mean = 1 ranks instead the mean
 *   of the chains' probabilities (the section's formula):
 *   sum_j exp(x_j[v] - lse_j), lse_j = ln sum_v exp(x_j[v]), fp32, summed in
 *   chain order (the 1/n_ept scale, which changes no ranking, left out); a
 *   chain row holding a NaN or +inf, or only -inf, makes every score NaN.
 *   Tokens whose mean probabilities differ by less than a few fp32 roundings
 *   may rank either way.  ept_mean = 0 is ppd_next_tree.
 *   tmpl_parent, tmpl_rank int32 [n_states][T_next] (device): the next tree of
 *   each state; node 0 is the root (parent -1), rank r >= 0 marks a candidate
 *   taking guess r at its depth, -1 a prompt node.
 * Outputs: next_parent, next_cand int32 [B][T_next] -- the state's template
 * with next_cand[0] = next_token[b], candidates filled, prompt nodes -1 (the
 * parent / cand_tokens of the next verification step); next_state [B] = k.
 * dev_status [B]: PPD_ERR_TREE (and outputs -1) when accept_len[b] < 1,
 * next_token[b] < 0, or template k is not a tree in topological order, has a
 * candidate below a prompt node, a candidate deeper than k or a rank >= K.
 * logits, parent, cand_tokens, path as for the verification step that just ran.
 * 1 <= K <= 16, K <= V; 1 <= n_ept <= 128; ept_mean 0 or 1; n_states <= 128;
 * T_next <= 512.
 * Workspace:
 * ppd_next_tree_workspace_bytes(B, n_states, K) bytes.
 */
size_t ppd_next_tree_workspace_bytes(int B, int n_states, int K);
ppd_status ppd_next_tree(const float *logits, const int32_t *parent, const int32_t *cand_tokens,
                         const int32_t *path, const int32_t *accept_len, const int32_t *next_token,
                         int B, int T, int V, int n_states, int T_next, const int32_t *tmpl_parent,
                         const int32_t *tmpl_rank, int K, int n_ept, int32_t *next_parent,
                         int32_t *next_cand, int32_t *next_state, int32_t *dev_status,
                         void *workspace, size_t ws_bytes,
                         void *stream);
ppd_status ppd_next_tree_ept(const float *logits, const int32_t *parent,
                             const int32_t *cand_tokens, const int32_t *path,
                             const int32_t *accept_len, const int32_t *next_token, int B, int T,
                             int V, int n_states, int T_next, const int32_t *tmpl_parent,
                             const int32_t *tmpl_rank, int K, int n_ept, int ept_mean,
                             int32_t *next_parent, int32_t *next_cand, int32_t *next_state,
                             int32_t *dev_status, void *workspace, size_t ws_bytes, void *stream);

/*
 * Node argmax without a workspace (no paper counterpart; an interface for
 * callers that cannot allocate device memory).  Same inputs, outputs, ranking
 * rule and stream behaviour as ppd_node_argmax, but the per-split partial maxima
 * live in a fixed 512 KiB array inside the library (a static __device__ object
 * that every GPU loading the library holds until the process exits), so the
 * call needs no scratch buffer.  It is meant for code that must not call
 * cudaMalloc or a caching allocator at this point: a plugin given only the
 * tensors it reads and writes, a real-time loop that forbids allocation after
 * start-up, or memory budgets that are fixed in advance.  The function itself
 * calls no allocating routine.
 *   - Size limit: B*T <= 65536 node rows; larger requests return
 *     PPD_ERR_UNSUPPORTED without enqueuing anything.
 *   - The first call on each device looks up the array's device address
 *     (cudaGetSymbolAddress, with that device current); make that first call
 *     before any stream capture that contains this entry point.
 *   - All calls share the array: calls whose kernels may overlap on the GPU
 *     (different streams without ordering) race and give undefined results.
 *     Nothing in the array needs to start at zero; each call rewrites what it reads.
 */
ppd_status ppd_node_argmax_noalloc(const float *logits, int B, int T, int V, int32_t *argmax_out,
                                   void *stream);

/*
 * Kernel launches one ppd_verify_step call (typical == 0) or
 * ppd_verify_step_typical call (typical != 0) enqueues for these sizes, with
 * a workspace of ppd_workspace_bytes(...) bytes and the whole GPU available.
 * No paper counterpart: it lets a caller or benchmark count the kernels of a
 * step without a profiler.  Returns -1 for sizes the step rejects.
 */
int ppd_verify_step_launches(int L, int B, int H, int T, int D, int V, int S_max, ppd_dtype dt,
                             int typical);

/*
 * The form a ppd_verify_step (or _typical) call takes for these sizes, with a
 * workspace of ppd_workspace_bytes(...) bytes and the whole GPU available
 * (no paper counterpart; for tests and benchmarks):
 *   0  B > 64: argmax, acceptance, attention and compaction as separate grids;
 *   1  an argmax grid, then the attention grid (which accepts and compacts);
 *   2  one attention grid whose spare warp per CTA also computes the argmax
 *      partial maxima while the K/V stream runs (chosen when the logits are
 *      at most 1/64 of the K/V bytes and form 3 does not fit);
 *   3  one attention grid whose softmax warps compute the argmax partial
 *      maxima before their first tile (chosen when the logits are at most
 *      128 KB per CTA of the attention grid).
 * Forms 2 and 3 fall back to form 1 when the cooperative launch cannot have
 * every CTA resident.  Returns -1 for sizes the step rejects.
 */
int ppd_verify_step_form(int L, int B, int H, int T, int D, int V, int S_max, ppd_dtype dt);

/*
 * Force the form of every later fused step of this process (B <= 64): 1, 2
 * or 3 as above, or -1 to return to the automatic choice.  The forms compute
 * the same results; this exists so that tests can cover each one at any size
 * and benchmarks can compare them (no paper counterpart).  Returns the
 * previous setting, or -2 (and changes nothing) for any other value.  Not
 * synchronised with steps already enqueued; set it while none is being
 * enqueued from another thread.
 */
int ppd_set_verify_step_form(int form);

/*
 * Diagnostics of the device-side timeout (no paper counterpart; for tests).
 * In the one-grid form (2) of every later fused step of this process, the
 * grid-wide wait for the argmax partials gives up after `limit_ns`
 * nanoseconds instead of 4 s (0 restores 4 s), and CTA `withhold_cta` never
 * publishes that its partials are ready (-1: every CTA does), so that a test
 * can make the wait run out: the step then reports PPD_ERR_TIMEOUT in
 * dev_status for every sequence, writes no cache row, and (as after any
 * timeout) its workspace must be zeroed before the next call.  Returns
 * PPD_ERR_INVALID_ARG for withhold_cta < -1.
 */
ppd_status ppd_debug_grid_wait(unsigned long long limit_ns, int withhold_cta);

/*
 * Name of the CUDA error behind the most recent PPD_ERR_CUDA returned in this
 * process ("cudaSuccess" if none; static string; diagnostics).
 */
const char *ppd_last_cuda_error(void);

/* Human-readable name of a status code (static string). */
const char *ppd_status_string(ppd_status s);

/*
 * Diagnostic (no paper counterpart): one 128 x N x 128 bf16 tensor-core product
 * through the same shared-memory layouts the attention kernel uses, so that a
 * test can check them against a plain matrix product.
 *   mode 0: d[128][N] = a[128][128] * b[N][128]^T   (both operands K-major)
 *   mode 1: d[128][N] = a[128][128]^T * b[128][N]   (a given [K][M], b given
 *           [K][N]: both operands M/N-major; b is written by threads)
 *   mode 2: as mode 1 with a given [K][64]; rows 64..127 of d repeat rows 0..63
 *   mode 3: d[128][N] = (a_hi + a_lo)[128][128] * b[128][N], a given [128][256]
 *           (columns 0..127 a_hi, 128..255 a_lo), held in tensor memory in the
 *           layout of the probability tile of the 65..128-token attention
 *           kernel and multiplied as two products; N <= 128
 * N in {16, 32, ..., 256}; a, b bf16 device pointers; d fp32 [128][N].
 */
ppd_status ppd_selftest_umma(const void *a, const void *b, float *d, int mode, int N,
                             void *stream);

#ifdef __cplusplus
}
#endif

#endif /* PPD_H */
