/*
 * dart.h -- C ABI of the GB300 (sm_103a) DARTree draft-tree construction path.
 *
 * The library builds the verification tree of one speculative-decoding round
 * from a block drafter's position-wise logits, following the paper "DARTree:
 * Speculative Diffusion Decoding with Autoregressive Draft Trees"
 * (arXiv 2608.13524):
 *   - Algorithm 1: for every depth d = 1..L, all retained prefixes S_{d-1}
 *     are scored in one batch by the correction head, every child is ranked
 *     by the Eq. 5 path score s_beta = sum_i log q~_i(u_i) + beta*d, the
 *     global top-W children form S_d, and their correction states are
 *     updated;
 *   - Sec. 4.3 / Lemma 1: the complete supertree S is pruned to the budget B
 *     with one global top-B (equal to best-first heap selection for
 *     beta <= 0), and flattened for tree-attention verification (Sec. 3.3).
 *
 * Correction head (the paper leaves its form open; this is the fallback head):
 *   h_c = RMSNorm(h_p + W_o . SiLU(W_i . [h_p ; E[t_c]]))   (no gain)
 * Corrected child distribution of a node with state h at depth d-1:
 *   z[v]  = (Dlog[d-1][v] + E[v] . h) / T'   (T' = T if T > 0, else 1)
 *   log q~[v] = min(z[v] - logsumexp_v z, 0)
 * The LM head is tied to the embedding table E.  The candidate set is the
 * whole vocabulary ("Full" in Appendix D) when cand_k = 0, or, as in
 * Algorithm 1 with K = cand_k (the paper's default K = 64, Sec. 5.1), the
 * set C_d = TopK(L_d^base, K) of the K largest drafter logits of position d
 * (ties: token asc), shared by every node of the depth; then v runs over
 * C_d only and q~ is renormalised over C_d (logsumexp over C_d).  Each node
 * keeps its top-k children by (log q~ desc, token asc), and S_d is the top-W
 * of those candidates by (score desc, parent slot asc, rank asc).  For
 * k >= W this equals the top-W over all children.  Candidates of score -inf
 * are never retained, so |S_d| <= min(W, |S_{d-1}| * k).
 *
 * Node ids: id = (depth-1)*W + rank within S_depth; ancestors always have
 * smaller ids.  Pruning keeps the top-B by (score desc, id asc).  Emission
 * lists the kept nodes in ascending id (a topological order).
 *
 * Conventions for every entry point:
 *   - all pointers are DEVICE pointers unless the name says _host;
 *   - `stream` is a cudaStream_t (NULL = legacy default stream); work is
 *     enqueued asynchronously and no call synchronises unless documented;
 *     with bf16 weights one GEMM of each depth runs on a second stream owned
 *     by the handle, forked from and joined back into `stream` by events
 *     within the same call (also when `stream` is being captured into a
 *     CUDA graph), so stream order as seen by the caller is unchanged;
 *   - return value: DART_OK or a negative dart_status; argument errors are
 *     detected on the host before anything is enqueued;
 *   - a handle must not be used from two streams or threads at once.
 */
#ifndef DART_H
#define DART_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct dart_handle dart_handle; /* opaque; owns its device workspace */

typedef enum {
    DART_OK = 0,
    DART_ERR_INVALID = -1,     /* bad argument, shape or pointer alignment */
    DART_ERR_CUDA = -2,        /* a CUDA runtime/driver call failed */
    DART_ERR_NOMEM = -3,       /* device or host allocation failed */
    DART_ERR_TIMEOUT = -4,     /* a device-side wait gave up (reported by dart_status_sync) */
    DART_ERR_STATE = -5,       /* call out of order (e.g. depth skipped) */
    DART_ERR_UNSUPPORTED = -6, /* device is not sm_103 / missing driver entry point */
    DART_ERR_BOUNDS = -7       /* debug builds only: a device index check failed (dart_status_sync) */
} dart_status;

typedef enum { DART_F32 = 0, DART_BF16 = 1 } dart_dtype;

/* Tuning switches of dart_config (every setting computes the same tree up
 * to the order of fp32 summation; DART_AUTO leaves the choice to the library). */
enum { DART_AUTO = 0, DART_ON = 1, DART_OFF = 2 };

/* Extra constructions a handle prepares for (dart_config.variants, bit set);
 * each allocates its own workspace at dart_init_head. */
enum {
    DART_VARIANT_CHAIN_DDTREE = 1, /* dart_build_chain_ddtree */
    DART_VARIANT_SEQ_HEAP = 2      /* dart_build_seq_heap */
};

/* Problem definition (Algorithm 1 inputs).
 *   V      vocabulary size, 1 <= V < 2^24, V >= k
 *   d      hidden size of the correction head, multiple of 64, 64 <= d <= 16384
 *   L      draft block length gamma (number of depths), 1 <= L, L*W <= 1024
 *   W      layer width (frontier size), 1 <= W <= 64
 *   k      per-node candidate count, 1 <= k <= 64, W*k <= 4096
 *   B      verification budget (non-root nodes kept), 1 <= B <= 1024
 *   nseq   independent sequences sharing the weights, nseq*W <= 256
 *   beta   depth bonus of Eq. 5, beta <= 0 (Lemma 1 precondition)
 *   temperature  T >= 0; T > 0 divides the logits by T, T = 0 is greedy
 *          scoring (no scaling)
 *   rms_eps      RMSNorm epsilon (> 0)
 *   pos_offset   position id of the root; a node at depth d gets pos_offset+d
 *   cand_k K of Algorithm 1: 0 scores every node over the full vocabulary;
 *          k <= cand_k <= min(V, 1024) scores it over C_d only
 * Tuning (DART_AUTO / DART_ON / DART_OFF; bf16 weights only, ignored for fp32):
 *   head_split         evaluate W_i . [h_p ; E[t_c]] as W_i[:, 0:d] . h_p plus
 *                      a row of the per-token table Q[t] = W_i[:, d:2d] . E[t]
 *                      (V*d floats of workspace, built at dart_init_head);
 *                      AUTO = ON.  OFF keeps no table (gather + full W_i GEMM)
 *   head_split_stream  with head_split: run the W_i[:, 0:d] GEMM on a second
 *                      stream beside the selection of the children; AUTO = ON
 *   lmhead_ctas_per_sm 1 or 2 LM-head CTAs per SM; 0 = 2 when both fit and
 *                      the weights are tiled or d <= 3072, else 1
 *   weights_tiled      the LM-head streams a copy of E re-laid as 128 x 64
 *                      tiles of 16 KB contiguous memory (made at
 *                      dart_init_head: ceil(V/128)*128*d bf16 of workspace)
 *                      instead of the caller's row-major E; AUTO = ON for
 *                      d <= 3072 with at most 16 nodes per depth (where it
 *                      was measured faster), else OFF
 *   head_weights_tiled the same for the head GEMMs' W_i (its first half with
 *                      head_split) and W_o (2*d*d or 3*d*d bf16); AUTO = OFF
 *   variants           bit set of DART_VARIANT_* (0: Algorithm 1 only); the
 *                      variants need cand_k = 0 and nseq <= 64, and the
 *                      chain's search keeps L * min(B, V) scores and tokens in
 *                      shared memory (DART_ERR_UNSUPPORTED beyond 227 KB)
 *   fused_round        fp32 weights: dart_build_tree runs the whole round
 *                      (every depth's scoring, merge, selection and head
 *                      update, then prune and emit) as one cooperative
 *                      kernel, one block per SM with grid-wide barriers,
 *                      instead of a graph of per-step launches.  Possible
 *                      with cand_k = 0, at most 32 nodes per depth
 *                      (nseq * W <= 32), L <= 32, L * W <= 256, k <= 32,
 *                      d <= 1024, V <= 65536 and the node states and
 *                      per-block scores within shared memory; AUTO = ON
 *                      where possible, ON = DART_ERR_UNSUPPORTED where not.
 *                      The depth-by-depth calls always take the per-step
 *                      launches (results agree within fp32 rounding)
 *   topk_bound         bf16 weights, cand_k = 0, V >= max(64, 2k): a
 *                      small kernel before each LM-head launch bounds every
 *                      node's k-th best score from below (its k-th best,
 *                      less an error bound, over the rows of largest drafter
 *                      logit in max(64, 2k) vocabulary chunks), and the
 *                      LM-head's top-k filter starts from that bound instead
 *                      of offering every logit of its first tiles to the
 *                      list merges.  The tree is unchanged.  AUTO = ON at
 *                      depths of more than 32 nodes (where it was measured
 *                      faster) */
typedef struct {
    int V, d, L, W, k, B, nseq;
    float beta, temperature, rms_eps;
    int pos_offset;
    int cand_k;
    int head_split, head_split_stream, lmhead_ctas_per_sm, weights_tiled, head_weights_tiled;
    int variants;
    int fused_round;
    int topk_bound;
} dart_config;

/* Emitted verification tree, caller-allocated, per sequence s:
 *   tokens [nseq][B]  token id of each kept node (-1 in unused rows)
 *   parents[nseq][B]  row of the parent in this array, -1 if the parent is
 *                     the root (the committed context), -2 in unused rows
 *   depths [nseq][B]  1..L (0 in unused rows)
 *   pos_ids[nseq][B]  pos_offset + depth (-1 in unused rows)
 *   scores [nseq][B]  Eq. 5 path score s_beta (-inf in unused rows)
 *   n_nodes[nseq]     number of used rows, min(B, |S|)
 *   mask   [nseq][B][ceil(B/64)]  ancestor bit mask: bit j of row i is set
 *                     iff row j is row i or one of its ancestors (the root /
 *                     context column is implicit and always visible); rows
 *                     beyond n_nodes are zero.  u64 words, bit j%64 of word j/64. */
typedef struct {
    int32_t *tokens, *parents, *depths, *pos_ids;
    float *scores;
    int32_t *n_nodes;
    uint64_t *mask;
} dart_tree_out;

/* Creates a handle for `cfg` and registers the head weights (Algorithm 1
 * input g, plus the tied LM head).  Weights are borrowed, never copied, and
 * must stay valid and unchanged for the handle's life:
 *   W_i [d][2d], W_o [d][d], E [V][d], row-major, of type `wdtype`
 *   (DART_BF16: bfloat16 with fp32 accumulation; DART_F32: float32 with
 *   fp32 arithmetic throughout).  Pointers must be 16-byte aligned.
 * Allocates the workspace for the worst case of cfg (synchronous
 * allocation).  With DART_BF16 weights it also computes on `stream` the
 * per-token table Q[t] = W_i[:, d:2d] . E[t] (fp32, V * d floats: 2.5 GB at
 * V = 151936, d = 4096), so that each state update adds one row of Q per
 * child instead of streaming the second half of W_i again; the call returns
 * after it is done (DART_ERR_TIMEOUT if a device-side wait of that GEMM gave
 * up).  Requires a compute capability 10.3 device (GB300).
 * On success *out receives the handle; on failure *out is NULL. */
int dart_init_head(dart_handle **out, const dart_config *cfg, int wdtype,
                   const void *W_i, const void *W_o, const void *E, void *stream);

/* Algorithm 1, one iteration: expands depth `depth` (1..L, in order; depth 1
 * restarts the round).  drafter_logits [nseq][L][V] float32 (row depth-1 is
 * read, 4-byte aligned), anchor_h [nseq][d] float32 = r_0 (16-byte aligned;
 * read at depth 1 only, may be NULL afterwards).  With cand_k > 0 the
 * candidate sets C_d of all L positions are taken at depth 1 from that
 * call's drafter_logits.  Out of order -> DART_ERR_STATE. */
int dart_expand_depth(dart_handle *h, int depth, const float *drafter_logits,
                      const float *anchor_h, void *stream);

/* Deferred pruning (Algorithm 1 final step, Lemma 1) and emission of the
 * verification tree after depth L was expanded; else DART_ERR_STATE. */
int dart_prune_and_emit(dart_handle *h, const dart_tree_out *out, void *stream);

/* The whole round: dart_expand_depth for 1..L, then dart_prune_and_emit.
 * Launched as one cached CUDA graph per distinct (inputs, outputs) pointer
 * set unless the stream is being captured by the caller.  The handle keeps
 * the graphs of its 8 most recently used pointer sets (least recently used
 * one destroyed first), so a caller rotating buffers does not grow memory. */
int dart_build_tree(dart_handle *h, const float *drafter_logits, const float *anchor_h,
                    const dart_tree_out *out, void *stream);

/* DARTree (fixed), the paper's first variant (Sec. 5.1): the supertree of
 * Algorithm 1 is itself the verification tree -- every retained node is
 * emitted, nothing is pruned (the paper's setting: W = 4 per depth, 64 nodes
 * over 16 depths).  Requires B >= sum_d |S_d| (at most L*W; else
 * DART_ERR_INVALID); otherwise as dart_build_tree, whose top-B then keeps
 * every node. */
int dart_build_tree_fixed(dart_handle *h, const float *drafter_logits, const float *anchor_h,
                          const dart_tree_out *out, void *stream);

/* Domino-chain + DDTree, the first alternative construction of Table 2
 * (Sec. 5.2): causal correction along ONE draft chain -- from r_0, at each
 * depth d the chain prefix's corrected distribution q~_d(. | y_<d) (full
 * vocabulary), its argmax y_d (log q~ desc, token asc) continuing the chain
 * -- then DDTree (Sec. 3.3) over those chain-conditioned distributions used
 * as position-wise marginals: best-first search over prefixes scored
 * s = sum_i log q~_i(u_i) + beta d (beta = 0 is DDTree's mass objective),
 * B pops.  Each pop takes the best "offer" -- every popped node (and the
 * root) offers its best child not yet taken -- by (score desc, popped node
 * asc, the root first).  The emitted rows are in pop order (parents first,
 * scores non-increasing); parents/depths/pos_ids/mask as for dart_build_tree.
 * Needs a handle made with DART_VARIANT_CHAIN_DDTREE in cfg.variants
 * (else DART_ERR_STATE).  Cost: L LM-head passes of one node per sequence,
 * the chain's L-1 head updates, a top-min(B, V) selection per depth and the
 * search.  Cached as a CUDA graph like dart_build_tree. */
int dart_build_chain_ddtree(dart_handle *h, const float *drafter_logits, const float *anchor_h,
                            const dart_tree_out *out, void *stream);

/* Sequential correction with heap, the second alternative construction of
 * Table 2 (Sec. 4.1): exact node-wise best-first search under the corrected
 * scores.  The root's children are scored at r_0; each of the B pops takes
 * the best offer as above -- but every node offers children from its OWN
 * corrected distribution -- and the popped prefix is then corrected before
 * the next pop: its state r(u_1..u_d) = g(r(u_<d), u_d) and the distribution
 * of its children q~_{d+1}(. | u_1..u_d) over the vocabulary (none at depth
 * L).  For beta <= 0 the result is the top-B of ALL prefixes by Eq. 5.
 * Emitted in pop order.  Needs DART_VARIANT_SEQ_HEAP in cfg.variants (else
 * DART_ERR_STATE).  Cost: up to B LM-head passes of one node per sequence,
 * one after another.  Cached as a CUDA graph like dart_build_tree. */
int dart_build_seq_heap(dart_handle *h, const float *drafter_logits, const float *anchor_h,
                        const dart_tree_out *out, void *stream);

/* Test hook after dart_build_chain_ddtree: the chain y [nseq][L] (int32)
 * and the log-sum-exp of each of its scaled-logit rows lse [nseq][L]
 * (float).  NULL outputs are skipped; DART_ERR_STATE after any other round. */
int dart_get_chain(dart_handle *h, int32_t *tok, float *lse, void *stream);

/* dart_build_tree on HOST buffers: copies drafter_logits_host [nseq][L][V]
 * and anchor_host [nseq][d] to handle-owned device staging, builds the tree
 * and copies it back into the host arrays of out_host (same layout as
 * dart_tree_out).  Synchronises `stream` before returning.  Pinned host
 * memory makes the copies asynchronous. */
int dart_build_tree_host(dart_handle *h, const float *drafter_logits_host,
                         const float *anchor_host, const dart_tree_out *out_host,
                         void *stream);

/* Test hook: copies S_depth of every sequence (after that depth was
 * expanded): tok / parent_slot / score [nseq][W] (rank order; parent_slot
 * -1 for children of the root, unused ranks tok -1, score -inf) and count
 * [nseq].  Any output pointer may be NULL. */
int dart_get_frontier(dart_handle *h, int depth, int32_t *tok, int32_t *parent_slot,
                      float *score, int32_t *count, void *stream);

/* Test hook: per expanded node of the most recent depth (rows
 * s*P + p, P = max |S_{depth-1}|): its k best children tok/logq [rows][k] and
 * the log-sum-exp of its scaled logits lse [rows].  *rows receives the row
 * count (host int).  NULL outputs are skipped. */
int dart_get_node_topk(dart_handle *h, int32_t *tok, float *logq, float *lse, int *rows,
                       void *stream);

/* Test hook: correction states r(u) [rows][d] float32 of the most recently
 * retained frontier (after the head update of depth < L).  *rows as above. */
int dart_get_states(dart_handle *h, float *states, int *rows, void *stream);

/* Synchronises `stream` and returns (then clears) the device status word:
 * DART_OK, DART_ERR_TIMEOUT if a kernel's bounded wait gave up, or (debug
 * builds) DART_ERR_BOUNDS if a data-dependent index failed its check. */
int dart_status_sync(dart_handle *h, void *stream);

/* Test hook of the fused round's grid barrier (handles with fused_round in
 * effect, else DART_ERR_STATE): two blocks wait at the handle's barrier for
 * a third that never comes, each gives up after limit_us microseconds
 * (1 <= limit_us <= 2000000) and sets the DART_ERR_TIMEOUT bit; nothing else
 * is touched.  The next dart_status_sync returns DART_ERR_TIMEOUT and resets
 * the barrier, after which the handle's rounds run normally again (before
 * it, dart_build_tree returns DART_ERR_STATE).  A fused round whose barrier
 * gave up on its own is reported and reset the same way. */
int dart_test_barrier_timeout(dart_handle *h, int limit_us, void *stream);

/* 1 in a library compiled with -DDART_DEBUG, else 0.  Debug builds check
 * every data-dependent index of the selection, emission, gather and heap
 * kernels (parent slots against the previous depth's count, token ids
 * against V, output positions against B) before it is used: a failing check
 * skips the access and sets a bit of the handle's status word, which the next
 * dart_status_sync returns as DART_ERR_BOUNDS; nothing traps. */
int dart_debug_build(void);

/* Test hook of the debug checks: one thread evaluates one failing index
 * check (an index equal to its bound) on `stream`, touching no memory but
 * the status word.  Debug builds: the next dart_status_sync returns
 * DART_ERR_BOUNDS; release builds: DART_OK (the checks compile away). */
int dart_test_bounds_report(dart_handle *h, void *stream);

/* Test hook for the failure path of the bounded device waits (no fault is
 * made): one CTA waits on an mbarrier that nothing completes, with the same
 * wait routine the kernels use but a limit of `limit_us` microseconds
 * (1 <= limit_us <= 2000000), gives up, sets the abort flag of its CTA and
 * the DART_ERR_TIMEOUT bit of the handle's status word; a second thread of
 * the CTA, waiting with the kernels' own 2 s limit on another such barrier,
 * must return as soon as it sees the abort flag.  No copy or MMA is in
 * flight.  elapsed_ns (optional, device int64 [2]) receives the time each of
 * the two waits took.  The next dart_status_sync returns DART_ERR_TIMEOUT. */
int dart_test_wait_timeout(dart_handle *h, int limit_us, int64_t *elapsed_ns, void *stream);

/* Profiling: when enabled, CUDA events bracket every LM-head scoring launch
 * (forces non-graph launches); dart_profile_read returns the summed device
 * time in ms and the launch count since the last read, and resets them. */
int dart_set_profiling(dart_handle *h, int enable);
int dart_profile_read(dart_handle *h, float *lmhead_ms, int *lmhead_launches);

/* Per-kind breakdown of the same profiling events (every launch is
 * bracketed while profiling is enabled).  Kinds: 0 LM-head scoring,
 * 1 merge + frontier select, 2 head-input gather, 3 head GEMM W_i
 * (W_i[:, 0:d] over the parents with the split first layer of bf16
 * weights), 4 SiLU + split, 5 head GEMM W_o, 6 residual + RMSNorm,
 * 7 depth-1 anchor preparation, 8 prune + emit, 9 candidate sets C_d
 * (cand_k > 0, once per round), 10 candidate scoring (cand_k > 0, per
 * depth), 11 gather of the per-token table row + SiLU + split (split first
 * layer), 12 top-K by value over a row of scaled logits (the best-first
 * constructions), 13 DDTree search, 14 one pop of the sequential search,
 * 15 its emission, 16 the fused small-problem round (fused_round: one
 * launch per round), 17 the early L2 prefetch of the next depth's first E
 * tiles (side stream), 18 the starting bound of the top-k filters
 * (topk_bound).  ms[i] / launches[i] receive the summed device time and
 * count of kind i for i < nkinds (nkinds <= 19); resets the events. */
int dart_profile_read_kinds(dart_handle *h, float *ms, int *launches, int nkinds);

/* Number of kernel launches one dart_build_tree enqueues for this handle. */
int dart_launches_per_round(dart_handle *h);

/* No-allocation variant of depth 1 (no counterpart in the paper: it exists
 * for callers that cannot allocate device memory while they run, e.g. a
 * serving engine that has reserved all free memory for its own pool, or a
 * path where cudaMalloc's implicit device synchronisation is not allowed).
 * It computes what dart_expand_depth(1) computes for every root -- the k best
 * children, their log q~ and the log-sum-exp over the full vocabulary, and
 * S_1 -- without a handle and without allocating:
 *   E [V][d] bf16 (16-byte aligned), drafter_logits [nseq][L][V] (row 0 is
 *   read), anchor_h [nseq][d] (16-byte aligned); outputs node_tok /
 *   node_logq [nseq][k], node_lse [nseq], front_tok / front_score [nseq][W]
 *   (rank order, unused ranks -1 / -inf), front_count [nseq].
 * Its scratch is one static 16 MiB device array that every GPU loading this
 * library keeps until the process exits.  Limits beyond dart_init_head's:
 * nseq <= 64, d <= 8192, full-vocabulary scoring only (cand_k = 0); other
 * problems return DART_ERR_INVALID before any
 * work is enqueued.  The first call on a device looks up the array's device
 * address (cudaGetSymbolAddress) and sets kernel attributes, so make that
 * first call before any stream capture.  Every call on a device shares the
 * array: calls that overlap on the GPU (other streams, other threads) race;
 * serialise them.  Device-side timeouts are not reported by the call
 * itself: dart_noalloc_status reads them afterwards. */
int dart_expand_root_noalloc(const dart_config *cfg, const void *E, const float *drafter_logits,
                             const float *anchor_h, int32_t *node_tok, float *node_logq, float *node_lse,
                             int32_t *front_tok, float *front_score, int32_t *front_count, void *stream);

/* After dart_expand_root_noalloc on the current device: synchronises
 * `stream` and returns DART_ERR_TIMEOUT if a device-side wait of the most
 * recent call gave up, else DART_OK (the status word lives in the static
 * array, at a fixed offset; nothing is allocated).  DART_ERR_STATE if no
 * call has been made on this device yet. */
int dart_noalloc_status(void *stream);

void dart_destroy(dart_handle *h);
const char *dart_status_string(int code);
int dart_version(void);

#ifdef __cplusplus
}
#endif
#endif /* DART_H */
