/*
 * treegraft.h - C ABI of the GB300 (sm_103a) library for the draft-tree
 * verify-and-grow step of TreeGraft (multi-drafter tree speculative decoding).
 *
 * General contract (all entry points):
 *  - Every pointer argument is a DEVICE pointer owned by the caller, unless
 *    stated otherwise.  The library never allocates device memory in these
 *    calls and never keeps a pointer after the call returns.
 *  - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *    stream).  Work is enqueued asynchronously on it; the call returns once
 *    the kernels are launched.
 *  - Arguments are validated on the host before anything is launched; an
 *    invalid call returns TG_ERR_INVALID_ARG or TG_ERR_UNSUPPORTED and
 *    launches nothing.  A failed launch returns TG_ERR_CUDA.
 *  - Conditions only visible on the device (a malformed parent[] array, a
 *    bounded wait that gave up) set bits in a per-device status word and the
 *    kernel returns early without touching memory out of range; read and
 *    clear that word with treegraft_last_device_status().
 *  - Trees are batched.  node_off[B+1] (int32) gives tree b the global node
 *    rows [node_off[b], node_off[b+1]); inside a tree, parent[] holds LOCAL
 *    ids with parent[0] = -1 and 0 <= parent[i] < i (parents before
 *    children, the order Algorithm 3 re-indexes the verification tree into).
 *    node_off[0] = 0 and node_off[B] = n_total (the trees cover the node
 *    rows exactly).  Every tree has at least one node (its root) and at
 *    most 256 nodes.  node_off lives on the device, so these conditions are
 *    checked there: a row that falls outside every tree's extent sets
 *    TG_ERR_DEVICE_TREE and takes no part in any tree's result.
 *  - bf16 data is IEEE bfloat16 (raw 16-bit patterns); all fp32/int32 data
 *    is native-endian.
 */
#ifndef TREEGRAFT_H
#define TREEGRAFT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  TG_OK = 0,
  TG_ERR_INVALID_ARG = 1,  /* null pointer, negative or inconsistent size */
  TG_ERR_UNSUPPORTED = 2,  /* valid but outside what the kernels implement */
  TG_ERR_CUDA = 3,         /* a CUDA runtime / driver call failed */
  TG_ERR_DEVICE_TREE = 4,  /* status bit: malformed tree seen on the device */
  TG_ERR_TIMEOUT = 8,      /* status bit: a bounded device wait gave up */
  TG_ERR_DEVICE_INDEX = 16 /* status bit: an index read from device memory was out of range */
} tg_status;

typedef enum { TG_BF16 = 0, TG_F32 = 1 } tg_dtype;

#define TG_MAX_TREE_NODES 256
#define TG_MAX_TOPK 32

/*
 * treegraft_tree_attn - ancestor-masked GQA tree attention.
 *
 * Paper: every draft-tree node attends over the committed prefix and its own
 * ancestors (Sec. 3.1 "verified efficiently ... through tree attention";
 * Algorithm 3 tree-attention mask: mask(u,v)=1 iff v is the root, an
 * ancestor of u, or u itself).  Used by the target's verification pass and
 * by the drafters' forward passes over the tree (Algorithms 1 and 2).
 *
 * For tree b, q-head h (kv-head h / G, G = Hq / Hkv) and local node u:
 *   keys J(u) = {0 .. P_b-1} U {P_b + v : mask(u, v)}
 *   o[u,h] = sum_{j in J(u)} softmax_j(scale * q[u,h] . k[j]) v[j]
 *   lse[u,h] = log sum_{j in J(u)} exp(scale * q[u,h] . k[j])   (natural log)
 *
 * q        bf16 [n_total, Hq, D], row-major (node, head, dim); 16-byte aligned.
 * k_cache,
 * v_cache  bf16 [B, Hkv, S_max, D]; slots [0, P_b) hold the committed prefix
 *          of sequence b, slots [P_b, P_b + n_b) the K/V of the tree's nodes
 *          in local node order (RoPE already applied by the caller).  Slots
 *          past P_b + n_b are never used and may hold anything (even NaN).
 * prefix_len int32 [B] (P_b >= 0, P_b + n_b <= S_max).
 * parent   int32 [n_total] local parent ids;  node_off int32 [B+1].
 * max_nodes  upper bound on n_b (<= 256); n_total = total node count.
 * D in {64, 128}; Hq % Hkv == 0, G = Hq / Hkv in {1, 2, 4, 8}.
 * scale    softmax scale; 0 selects D^-1/2.
 * out      bf16 [n_total, Hq, D];  lse_out fp32 [n_total, Hq] or NULL.
 * ws       scratch of treegraft_tree_attn_workspace_size(B, max_nodes, Hq,
 *          Hkv, D) bytes, 16-byte aligned, ZERO-FILLED before its first use;
 *          every call returns its counters to zero.  Calls sharing one ws
 *          must not overlap on the GPU.  Two plans use it:
 *          - small problems split the keys of a 128-row work unit over
 *            several thread blocks of a cooperative launch (the whole grid
 *            resident at once) that meet on counters in ws (a bounded wait,
 *            see treegraft_set_wait_budget: TG_ERR_TIMEOUT, never a hang)
 *            and combine their partial rows through ws;
 *          - batches whose whole units fill the GPU cut the keys of units
 *            well above the average share into chunks; each chunk writes
 *            its partial rows to ws and the last chunk of a unit to finish
 *            (a ticket in ws, no waiting) merges them.
 *          ws may be NULL (ws_bytes 0) when the sizes fill the GPU with
 *          whole units: every unit then stays whole.  A small problem
 *          without enough ws returns TG_ERR_INVALID_ARG.
 * Errors: TG_ERR_INVALID_ARG (null pointer, bad sizes, misaligned q/k/v),
 *   TG_ERR_UNSUPPORTED (D or G outside the list), TG_ERR_CUDA.  A malformed
 *   tree sets TG_ERR_DEVICE_TREE; its rows of `out` and `lse_out` are then
 *   undefined (computed with every tree slot masked).
 */
int treegraft_tree_attn(const void* q, const void* k_cache, const void* v_cache,
                        const int32_t* prefix_len, const int32_t* parent,
                        const int32_t* node_off, int B, int max_nodes, int n_total,
                        int Hq, int Hkv, int D, int S_max, float scale,
                        void* out, float* lse_out, void* ws, size_t ws_bytes, void* stream);

/*
 * treegraft_tree_attn_workspace_size - bytes of scratch treegraft_tree_attn
 * needs for these sizes (0 for invalid sizes).  Depends on no device state.
 */
size_t treegraft_tree_attn_workspace_size(int B, int max_nodes, int Hq, int Hkv, int D);

/*
 * treegraft_set_wait_budget - bound, in SM clock cycles, of the waits a
 * kernel makes on OTHER thread blocks: the split barrier of
 * treegraft_tree_attn, whose counters live in the caller's workspace.  A
 * wait that runs out raises TG_ERR_TIMEOUT in the device status word and
 * the kernel returns (that call's outputs are then undefined); the
 * counters are returned to zero, so the next call on the same workspace is
 * exact.  Waits inside one thread block (copies and tensor-core products)
 * keep their own fixed bound of about one second.  The budget applies to
 * the calls launched after it is set, process-wide.  cycles = 0 restores
 * the default (about one second at the GB300's maximum SM clock).  No
 * counterpart in the paper: this is a failure-detection control.
 * Errors: TG_ERR_INVALID_ARG for cycles < 0.
 */
int treegraft_set_wait_budget(int64_t cycles);

/*
 * treegraft_expand_topk - per-node log-softmax, top-k children, path scores.
 *
 * Paper: Top_m(l(v)) child tokens of a frontier node, edge score
 * p(u) = q(y | pi(v)) and cumulative score s(u) = s(v) p(u) (Sec. 3.1;
 * Algorithm 1, Algorithm 2 small and middle steps), kept in natural-log form.
 *
 * For logical row i (physical row r = row_idx ? row_idx[i] : i):
 *   lse[i]  = log sum_t exp(logits[r, t])
 *   tok[i,:] = the k token ids with the largest logits[r, t], ordered by
 *              (logit desc, token id asc) - exact on the input values
 *   logprob[i,j] = logits[r, tok[i,j]] - lse[i]
 *   score[i,j]   = parent_score[i] + logprob[i,j]
 * A row whose logits are all -inf gets lse = logprob = score = -inf and the
 * k lowest token ids.  Logits must be finite or -inf.
 *
 * logits   [logit_rows, ld] elements of `dtype` (TG_BF16 or TG_F32), row r
 *          at logits + r * ld; V <= ld; V <= 262144 (bf16) or 131072 (fp32);
 *          aligned to the element size (rows need no further alignment).
 * rows     number of logical rows (rows == 0 is a no-op).
 * row_idx  int32 [rows] of physical rows in [0, logit_rows), or NULL for
 *          rows 0..rows-1 (then rows <= logit_rows).
 * parent_score fp32 [rows].  1 <= k <= min(V, 32).
 * tok int32 [rows, k], logprob fp32 [rows, k], score fp32 [rows, k],
 * lse_out fp32 [rows] or NULL.
 * Errors: TG_ERR_INVALID_ARG, TG_ERR_UNSUPPORTED (V or k too large),
 *   TG_ERR_CUDA; an out-of-range row_idx sets TG_ERR_DEVICE_INDEX and that
 *   row's outputs are left unwritten.
 */
int treegraft_expand_topk(const void* logits, int dtype, int logit_rows, int V, int64_t ld,
                          int rows, const int32_t* row_idx, const float* parent_score, int k,
                          int32_t* tok, float* logprob, float* score, float* lse_out,
                          void* stream);

/*
 * treegraft_rescore_select - stronger-drafter rescoring + global top-N.
 *
 * Paper: at a middle-drafter step the candidate pool is
 * C_k = V(T_k) \ P_k (Sec. 3.2, expanded grafting-position selection); for
 * each non-root v in C_k the middle drafter replaces the edge score p(v),
 * s(root) stays 1 and s is recomputed; the grafting frontier is
 * F_k = Top_W(C_k, s) (Algorithm 2, middle-drafter branch).
 *
 * Per tree, with local ids and log-domain scores:
 *   edge[v]  = strong_lp[pa(v), token[v]]   if v != 0 and !visited[v]
 *            = weak_edge[v]                 if v != 0 and visited[v]
 *            = 0                            for the root
 *   score[0] = 0;  score[v] = fp32(score[pa(v)] + edge[v])   (in that order)
 *   selected = the N nodes of {v : !visited[v]} with the largest score,
 *              ordered by (score desc, node id asc); n_selected = their count
 *              (< N when the pool is smaller), remaining slots -1.
 * weak_edge fp32 [n_total]: stored edge log-probs p(v).
 * strong_lp fp32 [n_total, ld]: the stronger drafter's next-token log-probs;
 *   row node_off[b] + v is the distribution after local node v.  V <= ld.
 * parent, token int32 [n_total]; visited uint8 [n_total] (P_k, non-zero =
 * visited); node_off int32 [B+1].  1 <= N <= 256.
 * edge_out, score_out fp32 [n_total]; selected int32 [B, N] (local ids);
 * n_selected int32 [B].
 * Errors: TG_ERR_INVALID_ARG, TG_ERR_CUDA; malformed tree or token outside
 *   [0, V) sets TG_ERR_DEVICE_TREE / TG_ERR_DEVICE_INDEX and that tree's
 *   outputs are left unwritten.
 */
int treegraft_rescore_select(const float* weak_edge, const float* strong_lp, int V, int64_t ld,
                             const int32_t* parent, const int32_t* token,
                             const uint8_t* visited, const int32_t* node_off, int B,
                             int max_nodes, int n_total, int N, float* edge_out,
                             float* score_out, int32_t* selected, int32_t* n_selected,
                             void* stream);

/*
 * treegraft_accept_workspace_size - bytes of scratch treegraft_accept needs.
 */
size_t treegraft_accept_workspace_size(int B, int n_total);

/*
 * treegraft_graft_expand - expand the reselected grafting positions and
 * graft their children into the shared tree, non-destructively.
 *
 * Paper: the middle-drafter step of Sec. 3.2 / Algorithm 2 - after the
 * candidate pool is rescored and Top_W reselects grafting positions
 * (treegraft_rescore_select), each position v gets the drafter's top-m
 * next tokens as new children, appended to the tree without replacing any
 * existing node ("non-destructive grafting"), with edge score
 * p(u) = q(y | pi(v)) and path score s(u) = s(v) p(u) (log domain: sum).
 *
 * Trees use a capacity layout: tree b's nodes are rows [b*cap, b*cap + n)
 * of parent / token / edge / score, and the grafted children go to rows
 * b*cap + n + i*k + j for position slot i < N and rank j < k (the graft of
 * slot i is in slot order, its children in rank order).
 *   v      = selected[b*N + i]         (a LOCAL node id, 0 <= v < n)
 *   row    = logits row b*cap + v      (the drafter's next-token logits
 *                                       under the prefix ending at v)
 *   child j: parent = v, token = j-th largest logit of row (ties to the
 *            lower token), edge = logit - lse(row),
 *            score = fp32(score[b*cap + v] + edge)
 * logits   [logit_rows, ld] elements of dtype; rows must exist for every
 *          selected node.  V <= 262144 (bf16) / 131072 (fp32).
 * selected int32 [B, N], as treegraft_rescore_select writes it.  1 <= k <=
 *          min(V, 32); n + N*k <= cap.
 * parent, token int32 [B*cap]; edge, score fp32 [B*cap]: read at the
 *          selected rows, written at the appended rows.
 * Errors: TG_ERR_INVALID_ARG, TG_ERR_UNSUPPORTED, TG_ERR_CUDA.  A selected
 *   id outside [0, n), or a logits row past logit_rows, sets
 *   TG_ERR_DEVICE_INDEX and that slot's children are left unwritten.
 */
int treegraft_graft_expand(const void* logits, int dtype, int logit_rows, int V, int64_t ld,
                           int B, int N, const int32_t* selected, int k, int cap, int n,
                           int32_t* parent, int32_t* token, float* edge, float* score,
                           void* stream);

/*
 * treegraft_accept - greedy longest-accepted-path walk (temperature 0).
 *
 * Paper: verification of the pruned tree with the target model and the
 * standard rule (Algorithm 1/2, final step; Sec. 3.2 "Distribution
 * preservation"), at temperature 0 (Appendix E) - greedy matching.
 *
 * Per tree:  am[v] = argmax_t target[v, t] (lowest t on ties);
 *   full[0] = true; full[v] = full[pa(v)] and token[v] == am[pa(v)];
 *   a* = the full node of greatest depth, lowest id on ties;
 *   accept_len = depth(a*) (accepted draft tokens, root excluded);
 *   path = root-first local ids of the root..a* chain, padded with -1 to
 *   path_cap; bonus = am[a*] (the target's next token after a*).
 * target_logits [n_total, ld] of `dtype`, aligned to the element size; row
 * node_off[b] + v belongs to local node v.  token int32 [n_total] (token[root] ignored).
 * path int32 [B, path_cap] (path_cap >= 1); accept_len, bonus int32 [B].
 * ws       scratch of treegraft_accept_workspace_size(B, n_total) bytes,
 *          16-byte aligned, ZERO-FILLED before its first use with this
 *          function; each call on well-formed trees leaves it all zero
 *          again, so one ws serves later calls of any B and n_total that
 *          fit it.  Calls sharing one ws must not overlap on the GPU.
 * Errors: TG_ERR_INVALID_ARG, TG_ERR_UNSUPPORTED (V > 262144 for bf16 or
 *   > 131072 for fp32), TG_ERR_CUDA;
 *   a malformed tree sets TG_ERR_DEVICE_TREE, a path longer than path_cap
 *   sets TG_ERR_DEVICE_INDEX (that tree's outputs are then left unwritten).
 */
int treegraft_accept(const void* target_logits, int dtype, int V, int64_t ld,
                     const int32_t* token, const int32_t* parent, const int32_t* node_off,
                     int B, int max_nodes, int n_total, int path_cap, int32_t* path,
                     int32_t* accept_len, int32_t* bonus, void* ws, size_t ws_bytes,
                     void* stream);

/*
 * treegraft_accept_noalloc - treegraft_accept for callers that cannot
 * allocate device memory.
 *
 * The paper has no counterpart: this is a library convenience.  Some callers
 * cannot obtain a scratch buffer - a plugin that an inference engine hands
 * only its inputs and outputs, or code running where every device
 * allocation must go through a pool it cannot reach.  This variant takes no
 * `ws` and allocates nothing: its scratch lives in a fixed array inside the
 * library, so every GPU that loads the library holds about 272 KB for it
 * until the process exits.
 *
 * Arguments, outputs and results are those of treegraft_accept (without ws
 * and ws_bytes).  Limits of the fixed array: n_total <= TG_NOALLOC_MAX_NODES
 * and B <= TG_NOALLOC_MAX_TREES; larger calls return TG_ERR_UNSUPPORTED and
 * launch nothing.
 * The first call on a device looks up the array's device address
 * (cudaGetSymbolAddress); make that first call before any stream capture.
 * The address is kept for the life of the process: after cudaDeviceReset
 * (or anything else that destroys the device's primary context) it is stale,
 * so this library must not be used across such a reset.  The same holds for
 * the device status word that every call of this header writes.
 * All calls on a device share the one array: calls that overlap on the GPU
 * (other streams, other host threads) race and give wrong results; order
 * them on one stream.  Each call clears the counters it needs on `stream`
 * (cudaMemsetAsync) before its kernel runs.
 */
#define TG_NOALLOC_MAX_NODES 65536
#define TG_NOALLOC_MAX_TREES 4096
int treegraft_accept_noalloc(const void* target_logits, int dtype, int V, int64_t ld,
                             const int32_t* token, const int32_t* parent,
                             const int32_t* node_off, int B, int max_nodes, int n_total,
                             int path_cap, int32_t* path, int32_t* accept_len, int32_t* bonus,
                             void* stream);

/*
 * treegraft_global_prune - global score-based pruning with ancestor closure,
 * and the verification buffers of the pruned tree.
 *
 * Paper: Algorithm 3 (GlobalPrune, called by Algorithms 1 and 2 before
 * target verification).  Per tree, with M = budget + 1 (the root is the
 * extra node): a tree of at most M nodes is kept whole; otherwise the
 * non-root nodes are ranked by (score desc, depth asc, id asc) and, from
 * K = {root}, each ranked node's chain up to the first node in K is added
 * whole when |K| + |chain| <= M, stopping once |K| = M.  Kept nodes are
 * re-indexed in their original order (parents stay before children).
 *
 * score    fp32 [n_total] path scores (log domain, larger is better; the
 *          root's is ignored).  Finite or -inf.
 * parent   int32 [n_total] local parent ids; node_off int32 [B+1]; trees of
 *          1..TG_MAX_PRUNE_NODES nodes, n_total <= B * max_nodes.
 * budget   B_ver >= 1 with budget + 1 <= TG_MAX_TREE_NODES (the pruned
 *          tree must fit treegraft_tree_attn).
 * Outputs, with stride Mo = min(budget + 1, max_nodes) per tree:
 *   kept       int32 [B, Mo]  old local ids in new order, -1 padded;
 *   n_kept     int32 [B];
 *   new_parent int32 [B, Mo]  parent in new ids (-1 for the root and pad);
 *   position   int32 [B, Mo]  position id = depth (-1 pad);
 *   mask       uint32 [B, Mo, ceil(Mo / 32)]  row i bit j set iff new node
 *              j is the root, an ancestor of i, or i itself (Algorithm 3
 *              mask); rows past n_kept are zero;
 *   paths      int32 [B, Mo, path_cap]  root-to-leaf retrieval paths in new
 *              ids, one row per leaf in ascending new id, root first, -1
 *              padded; rows past n_paths are -1;
 *   n_paths    int32 [B].
 * Errors: TG_ERR_INVALID_ARG, TG_ERR_UNSUPPORTED (max_nodes >
 *   TG_MAX_PRUNE_NODES), TG_ERR_CUDA; a malformed tree sets
 *   TG_ERR_DEVICE_TREE (its outputs left unwritten); a path longer than
 *   path_cap sets TG_ERR_DEVICE_INDEX (the path is cut at path_cap).
 */
#define TG_MAX_PRUNE_NODES 1024
int treegraft_global_prune(const float* score, const int32_t* parent, const int32_t* node_off,
                           int B, int max_nodes, int n_total, int budget, int path_cap,
                           int32_t* kept, int32_t* n_kept, int32_t* new_parent,
                           int32_t* position, uint32_t* mask, int32_t* paths, int32_t* n_paths,
                           void* stream);

/*
 * treegraft_grow_step - one drafting step of the shared draft tree.
 *
 * Paper: Algorithm 2 (TreeGraft shared-tree construction with grafting), one
 * iteration k; with small-drafter steps only it is Algorithm 1.  Scores are
 * log-probabilities (s(root) = 0, s(u) = fp32(s(v) + p(u)), p(u) the
 * drafter's natural-log probability of u's token after the prefix ending at
 * v); Top_W ranks nodes by (s desc, id asc), Top_m tokens by (logit desc,
 * token asc).
 *   mode 0 (small drafter): candidate pool C = N_k, the nodes the previous
 *     step made; F = Top_W(C, s); every v in F gets the m best tokens of its
 *     row of `logits` (the small drafter's table) as children.
 *   mode 1 (middle drafter): C = V(T) \ P; the row of every v in C is
 *     log-softmax normalised and its log-sum-exp cached in lse_mid[v]; every
 *     non-root v in C is rescored, p(v) = l[pa(v), token(v)] - lse_mid[pa(v)]
 *     (its parent's middle-drafter row, visited or not), and s is recomputed
 *     root-first; F = Top_W(C, s); every v in F gets the m best tokens of its
 *     row.  Then P = P u C.
 * Children are appended after the last node, in frontier order then child
 * rank, without replacing any node (a duplicate token is a new sibling).
 *
 * Trees: B trees of capacity `cap` (1 <= cap <= TG_MAX_GROW_NODES); tree b
 * owns rows [b * cap, (b + 1) * cap) of parent, token, edge, score, lse_mid
 * and of the logit table, with local ids.  All trees grow in lock step with
 * one schedule, so the sizes are the caller's (host) numbers:
 *   n        nodes per tree before the step (>= 1: the root alone is n = 1,
 *            parent[0] = -1, score[0] = 0, edge[0] = 0);
 *   pool_lo  the pool is [pool_lo, n).  mode 0: the first node the previous
 *            step made (0 at the first step, where N_1 = {root}).  mode 1:
 *            |P|, the node count when the last middle step ran (0 if none) -
 *            P is always the prefix [0, |P|) of the ids, because a middle
 *            step visits every node that exists and nodes are only appended.
 * After the step each tree has n + min(W, n - pool_lo) * m nodes (must be
 * <= cap), the next small step pools [n, that), and after a middle step
 * |P| = n.
 * logits   [B * cap, ld] bf16 or fp32: row b * cap + v is the drafter's
 *          next-token logits after node v of tree b (its forward over the
 *          tree); V <= ld columns used.
 * parent, token int32, edge, score fp32 [B * cap]: the tree, updated in place
 *          (the pool's edge and score are rewritten by a middle step).
 * lse_mid  fp32 [B * cap]: log-sum-exp of the middle drafter's rows, written
 *          for the pool by a middle step and read for visited parents; may
 *          be NULL if mode is 0.
 * frontier int32 [B, W]: F in rank order, -1 padded.
 * ws       scratch of treegraft_grow_workspace_size(B, cap, m) bytes,
 *          16-byte aligned; no initial contents required.
 * Errors: TG_ERR_INVALID_ARG (null pointer, sizes, capacity overflow),
 * TG_ERR_UNSUPPORTED (cap > TG_MAX_GROW_NODES, m > TG_MAX_TOPK, vocabulary
 * above 262144 bf16 / 131072 fp32), TG_ERR_CUDA.  A malformed parent array
 * sets TG_ERR_DEVICE_TREE, a token outside [0, V) in a middle pool sets
 * TG_ERR_DEVICE_INDEX; the step's outputs are then undefined.
 */
#define TG_MAX_GROW_NODES 1024
size_t treegraft_grow_workspace_size(int B, int cap, int m);
int treegraft_grow_step(int mode, const void* logits, int dtype, int V, int64_t ld, int B, int cap,
                        int n, int pool_lo, int W, int m, int32_t* parent, int32_t* token,
                        float* edge, float* score, float* lse_mid, int32_t* frontier, void* ws,
                        size_t ws_bytes, void* stream);

/*
 * treegraft_accept_sample - verification at temperature T > 0: the tree
 * rejection-sampling rule behind the distribution preservation of Sec. 3.2
 * (Algorithms 1 and 2, verification step), for children that are
 * deterministic proposals.  At node v (from the root) with p =
 * softmax(target_logits[v] / T) and the residual r = p, v's children are
 * visited in ascending node id; child c with token x is accepted iff
 * u[c, 0] * sum(r) < r(x) (r holding p minus the tokens of the children
 * rejected before c, so a child repeating an earlier sibling's token is
 * never accepted); the walk moves to the first accepted child.  At the node
 * a* where every child is rejected (or a leaf) the bonus token is drawn from
 * r / sum(r) by inversion: the first token t whose cumulative residual mass
 * exceeds u[a*, 1] * sum(r).  Each emitted token then follows p exactly.
 *
 * Trees, target_logits, path, accept_len and path_cap are as in
 * treegraft_accept.  u: fp32 [n_total, 2] uniforms in [0, 1) on the
 * device, drawn by the caller (u[c, 0] decides child c, u[v, 1] the bonus
 * draw at v).  temperature > 0 (fp32 must be able to hold log2(e) / T).
 * ws: treegraft_accept_sample_workspace_size(B, n_total) bytes, 16-byte
 * aligned, ZEROED before its first use (per-node flags and candidates,
 * per-tree tickets); each call on well-formed input leaves it all zero
 * again, so one ws serves later calls of any B and n_total that fit it.
 * One launch: per node row, the masses 2^((l - max) log2(e) / T)
 * in 44-bit fixed point (exact, order-free sums), every child's decision
 * and the bonus draw the row would give if the walk ended there; the CTA
 * that finishes a tree's rows walks it.  The masses carry the rounding of
 * the exponential and of the fixed point, so a draw within about 1e-7 of
 * a threshold may fall either way.
 * Errors: TG_ERR_INVALID_ARG, TG_ERR_UNSUPPORTED (V too large, B > 65535,
 * T too small), TG_ERR_CUDA; a malformed tree sets TG_ERR_DEVICE_TREE and a
 * token outside [0, V) or a path longer than path_cap TG_ERR_DEVICE_INDEX
 * (that tree's outputs are then undefined).
 */
size_t treegraft_accept_sample_workspace_size(int B, int n_total);
int treegraft_accept_sample(const void* target_logits, int dtype, int V, int64_t ld,
                            float temperature, const int32_t* token, const int32_t* parent,
                            const int32_t* node_off, int B, int max_nodes, int n_total,
                            const float* u, int path_cap, int32_t* path, int32_t* accept_len,
                            int32_t* bonus, void* ws, size_t ws_bytes, void* stream);

/*
 * n-gram small drafter (Appendix, "n-gram small drafter"; the small drafter
 * of Algorithm 2).  A training-free lookup: at prefill the target's top
 * m_cache next-token candidates and their log-probabilities are cached at
 * every prompt position, and an n-gram index is built over the prompt; at a
 * small-drafter step the suffix of the prefix at tree node v is matched in
 * the prompt with the longest n-gram that occurs (max_n tokens, then one
 * fewer, ... down to one), at the n-gram's latest occurrence, and the
 * candidates cached at the matched position become v's children, their
 * cached log-probabilities the edge scores p(u).  With no match at any
 * length the position of the prompt's most frequent token (ties to the
 * lower token id; its latest occurrence) is used.
 *
 * Prompts are packed: `tokens` int32 [n_tokens], sequence b owns positions
 * [seq_off[b], seq_off[b + 1]) (seq_off int32 [B + 1] on the device,
 * seq_off[0] = 0, strictly increasing: every prompt non-empty,
 * seq_off[B] = n_tokens).  Tree b of a draft or grow call belongs to prompt b.
 * The prefix at node v is the committed text followed by the tokens of the
 * non-root nodes on the path root -> v: the committed text's last max_n
 * tokens are ctx[b * max_n + 0 .. ctx_len[b]) (int32 [B, max_n] and [B] on
 * the device, oldest first; its last token is the root's, so token[root] is
 * not read; 0 <= ctx_len[b] <= max_n).  Only the prompt is indexed (its
 * positions are the ones with cached candidates); a match lies wholly
 * inside one prompt.
 *
 * treegraft_ngram_index_bytes: bytes of the index for (B, n_tokens,
 *   max_n); 0 for an invalid or unsupported shape.
 * treegraft_ngram_build: build the index into `index` (caller-owned device
 *   buffer, 16-byte aligned, no initial contents required; it keeps its own
 *   copy of the tokens).  Four launches.  A malformed seq_off sets
 *   TG_ERR_DEVICE_INDEX (the index is then unusable).
 * treegraft_ngram_cache: the prefill cache from the prefill logits [rows,
 *   ld] (row i = the target's next-token logits after packed position i, so
 *   rows = n_tokens): cache_tok int32 [rows, m_cache] by (logit desc, token
 *   asc), cache_lp fp32 [rows, m_cache] = fp32(logit - lse).  One
 *   expand_topk launch.
 * treegraft_ngram_draft: the drafter's expansion of arbitrary tree nodes:
 *   rows int32 [R] (device) = b * cap + v; parent, token int32 [B * cap]
 *   (tree b at rows [b * cap, (b + 1) * cap), local ids, parents before
 *   children); outputs tok int32, logprob, score fp32 [R, m] with score =
 *   fp32(parent_score[r] + logprob) for the first m <= m_cache cached
 *   candidates; match_pos int32 [R] (position within its prompt) and
 *   match_n int32 [R] (the order matched, 0 for the fallback) may be NULL.
 *   One launch, one warp per row.
 * treegraft_ngram_grow_step: one small-drafter step of Algorithm 2 with this
 *   drafter on B trees of capacity cap (the tree layout, n, pool_lo, W, m
 *   and frontier of treegraft_grow_step with mode 0): F = Top_W of the pool
 *   [pool_lo, n) by (s desc, id asc), each node of F gets the first m
 *   candidates of its lookup as children, appended at n, n + 1, ... in
 *   frontier order then candidate rank, edge = the cached log-probability,
 *   score = fp32(s(v) + edge).  One launch, one CTA per tree.
 * Errors: TG_ERR_INVALID_ARG (null pointer, sizes, m > m_cache, a small
 *   index buffer, capacity overflow), TG_ERR_UNSUPPORTED (max_n >
 *   TG_NGRAM_MAX_N, n_tokens > TG_NGRAM_MAX_TOKENS, m_cache > TG_MAX_TOPK,
 *   cap > TG_MAX_GROW_NODES), TG_ERR_CUDA.  On the device: a malformed tree
 *   sets TG_ERR_DEVICE_TREE, a row outside [0, B * cap), a ctx_len outside
 *   [0, max_n] or a prompt with no fallback position sets
 *   TG_ERR_DEVICE_INDEX; the affected outputs are then undefined.
 */
#define TG_NGRAM_MAX_N 8
#define TG_NGRAM_MAX_TOKENS (1 << 26)
size_t treegraft_ngram_index_bytes(int B, int n_tokens, int max_n);
int treegraft_ngram_build(const int32_t* tokens, const int32_t* seq_off, int B, int n_tokens,
                          int max_n, void* index, size_t index_bytes, void* stream);
int treegraft_ngram_cache(const void* logits, int dtype, int rows, int V, int64_t ld, int m_cache,
                          int32_t* cache_tok, float* cache_lp, void* stream);
int treegraft_ngram_draft(const void* index, size_t index_bytes, int B, int n_tokens, int max_n,
                          const int32_t* cache_tok, const float* cache_lp, int m_cache,
                          const int32_t* ctx, const int32_t* ctx_len, const int32_t* parent,
                          const int32_t* token, int cap, const int32_t* rows, int R,
                          const float* parent_score, int m, int32_t* tok, float* logprob,
                          float* score, int32_t* match_pos, int32_t* match_n, void* stream);
int treegraft_ngram_grow_step(const void* index, size_t index_bytes, int B, int n_tokens,
                              int max_n, const int32_t* cache_tok, const float* cache_lp,
                              int m_cache, const int32_t* ctx, const int32_t* ctx_len, int cap,
                              int n, int pool_lo, int W, int m, int32_t* parent, int32_t* token,
                              float* edge, float* score, int32_t* frontier, void* stream);

/*
 * treegraft_last_device_status - synchronise `stream`, return the OR of the
 * device status bits raised since the last call on the current device
 * (TG_OK if none), and clear them.  Returns TG_ERR_CUDA if the
 * synchronisation itself fails.
 */
int treegraft_last_device_status(void* stream);

/* Human-readable name of a status value (static string). */
const char* treegraft_status_string(int status);

#ifdef __cplusplus
}
#endif

#endif /* TREEGRAFT_H */
