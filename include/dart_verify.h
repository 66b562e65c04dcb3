/*
 * dart_verify.h -- tree-attention verification consumer of the emitted draft
 * tree (GB300, sm_103a).
 *
 * Sec. 3.3 of the paper ("Tree Verification and DDTree") flattens the draft
 * tree and verifies every branch in ONE target forward pass: each tree node
 * attends to the verified context and to the tokens on its own root-to-node
 * path, and nothing else.  Sec. 4.3 (after Lemma 1) hands the pruned tree to
 * exactly that pass.  The target model is not available here, so this
 * library provides the part of the pass that the tree changes -- one
 * attention layer over [context ; tree] with the tree mask and the tree
 * position ids -- on synthetic Q / K / V:
 *
 *   for every sequence s, tree row i < n_nodes[s] and query head h
 *   (kv head g = h / (Hq / Hkv)):
 *     q  = RoPE(Q[s,i,h], pos_ids[s,i])
 *     keys   = { Kc[s,c,g] : 0 <= c < C }                 (context, all visible)
 *            u { RoPE(Kt[s,j,g], pos_ids[s,j]) : bit j of mask[s,i] }
 *     values = the matching rows of Vc[s,:,g] and Vt[s,:,g]
 *     out[s,i,h] = softmax(scale * q . keys) . values
 *   rows i >= n_nodes[s] are written as zeros.
 *
 * RoPE is the rotate-half form: for 0 <= t < dh/2, with
 * inv_freq_t = rope_theta^(-2t/dh) and angle = pos * inv_freq_t,
 *   y[t]        = x[t] cos(angle) - x[t + dh/2] sin(angle)
 *   y[t + dh/2] = x[t + dh/2] cos(angle) + x[t] sin(angle).
 * The context keys are a KV cache: already rotated at their positions.
 *
 * The tree arrays are the ones dart_prune_and_emit writes (include/dart.h):
 * pos_ids [nseq][B] (pos_offset + depth), the ancestor bitmask
 * [nseq][B][ceil(B/64)] (bit j of row i set iff j is i or an ancestor of i)
 * and n_nodes [nseq].  dart_ancestor_mask builds the same mask from a parent
 * array, for trees that come from elsewhere.
 *
 * Conventions: DEVICE pointers, asynchronous on `stream` (a cudaStream_t,
 * NULL = legacy default stream), return 0 or a negative dart_status code of
 * include/dart.h; argument errors are detected on the host before anything
 * is enqueued.
 */
#ifndef DART_VERIFY_H
#define DART_VERIFY_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct {
    int nseq;         /* independent sequences, >= 1 */
    int B;            /* tree rows per sequence, 1..1024 */
    int C;            /* context keys per sequence, >= 0 */
    int Hq, Hkv;      /* query / key-value heads; Hq / Hkv in {1, 2, 4, 8, 16} */
    int dh;           /* head dimension; 128 */
    float rope_theta; /* RoPE base, > 1 */
    float scale;      /* softmax scale, e.g. 1 / sqrt(dh); > 0 */
} dart_attn_config;

/* Device workspace (bytes) dart_tree_attention needs for `cfg`; 0 on an
 * invalid configuration. */
size_t dart_tree_attention_workspace(const dart_attn_config *cfg);

/* One tree-attention layer (see above).  Layouts, all row-major bf16 unless
 * stated, innermost dimension last:
 *   q       [nseq][B][Hq][dh]    queries of the tree rows, not rotated
 *   k_tree  [nseq][B][Hkv][dh]   keys of the tree rows, not rotated
 *   v_tree  [nseq][B][Hkv][dh]
 *   k_ctx   [nseq][C][Hkv][dh]   rotated context keys (may be NULL if C = 0)
 *   v_ctx   [nseq][C][Hkv][dh]   (may be NULL if C = 0)
 *   pos_ids [nseq][B] int32, mask [nseq][B][ceil(B/64)] uint64,
 *   n_nodes [nseq] int32 (0 <= n_nodes <= B)
 *   out     [nseq][B][Hq][dh] fp32 (written; rows >= n_nodes are zero)
 *   workspace: device memory of dart_tree_attention_workspace(cfg) bytes,
 *   256-byte aligned, owned by the caller, used by this call only until
 *   the stream reaches its end (no state is kept between calls).
 * Every tensor pointer must be 16-byte aligned.  Mask bits at or beyond
 * n_nodes are ignored.  Returns DART_ERR_INVALID for a bad configuration,
 * a NULL or misaligned pointer or a too small workspace,
 * DART_ERR_UNSUPPORTED when the device cannot run the kernel (not sm_103a,
 * too little shared memory), DART_ERR_CUDA on a launch error.  A bounded
 * device wait that gives up sets bit 1 (value 1) of *status (a device int
 * the caller zeroes; may be NULL) and leaves `out` unspecified. */
int dart_tree_attention(const dart_attn_config *cfg, const void *q, const void *k_tree, const void *v_tree,
                        const void *k_ctx, const void *v_ctx, const int32_t *pos_ids, const uint64_t *mask,
                        const int32_t *n_nodes, float *out, void *workspace, size_t workspace_bytes,
                        int *status, void *stream);

/* dart_tree_attention followed by a synchronisation of `stream`; *ms_rope
 * and *ms_attn receive the device time of the RoPE pre-pass and of the
 * attention kernel (CUDA events recorded around each launch on `stream`).
 * For benchmarking; same arguments and errors, plus DART_ERR_INVALID for a
 * NULL ms_rope / ms_attn. */
int dart_tree_attention_timed(const dart_attn_config *cfg, const void *q, const void *k_tree, const void *v_tree,
                              const void *k_ctx, const void *v_ctx, const int32_t *pos_ids, const uint64_t *mask,
                              const int32_t *n_nodes, float *out, void *workspace, size_t workspace_bytes,
                              int *status, float *ms_rope, float *ms_attn, void *stream);

/* Ancestor bitmask of flattened trees given by parent indices:
 * parents [nseq][B] int32 with -1 for a child of the root and
 * 0 <= parents[i] < i otherwise (a topological order, as emitted);
 * rows i >= n_nodes[s] and bits j >= n_nodes[s] are zero.  A parent index
 * outside [-1, i) ends the walk there (the row keeps the bits found so far).
 * mask [nseq][B][ceil(B/64)] uint64 is written.  Returns DART_ERR_INVALID
 * for nseq < 1, B outside 1..1024 or a NULL pointer. */
int dart_ancestor_mask(const int32_t *parents, const int32_t *n_nodes, int nseq, int B, uint64_t *mask,
                       void *stream);

#ifdef __cplusplus
}
#endif

#endif /* DART_VERIFY_H */
