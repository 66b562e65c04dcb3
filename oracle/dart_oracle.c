/*
 * DARTree draft-tree construction: plain fp64 CPU oracle.
 *
 * TEST INFRASTRUCTURE ONLY.  The tests, the smoke check and the benchmark's
 * CPU-baseline leg load this library; the product (CUDA) path never does and
 * shares no code with it.  Everything here is written to be read against the
 * paper, not to be fast: fp64 throughout, one straightforward loop per
 * formula, no blocking or fusion.  OpenMP only splits independent vocabulary
 * rows / output features across threads; every reduction that could depend
 * on the thread count (log-sum-exp, top-k, sorting) runs serially.
 *
 * What it computes (paper: "DARTree: Speculative Diffusion Decoding with
 * Autoregressive Draft Trees", arXiv 2608.13524):
 *   - Algorithm 1 (depth-wise fixed-width supertree construction) with a
 *     per-node top-k, over either the full vocabulary (Appendix D, "Full")
 *     or the candidate set C_d = TopK(L_d^base, K) of Algorithm 1 (cand_k =
 *     K > 0; the paper's default is K = 64, Sec. 5.1);
 *   - the path score of Eq. 5, s_beta(u_{1:d}) = sum_i log q~_i(u_i) + beta d;
 *   - deferred pruning, T = TopB_{u in S} s_beta(u) (Algorithm 1, final step);
 *   - the best-first heap of Sec. 4.3 / Lemma 1 (used to check that the top-B
 *     selection equals heap selection when beta <= 0);
 *   - flattening into the verification tree with an ancestor mask
 *     (Sec. 3.3, tree verification).
 * Readings where the paper is silent:
 *   - correction head g = fallback head
 *       h_c = RMSNorm(h_p + W_o SiLU(W_i [h_p ; E[t_c]])),  RMSNorm without gain;
 *   - corrected child distribution of a node with state h at depth d-1:
 *       z[v] = (Dlog[d-1][v] + E[v] . h) / T'   (T' = T if T > 0 else 1),
 *       log q~[v] = min(z[v] - logsumexp(z), 0)  (clamp keeps Lemma 1 exact),
 *     the log-sum-exp running over the vocabulary, or over C_d when the
 *     candidate set is restricted (q~ renormalised over C_d: Algorithm 1
 *     evaluates g only on C_d, so tokens outside C_d have no probability);
 *   - C_d = the K tokens of largest drafter logit Dlog[d-1][v] (ties: token
 *     asc), the same for every node of the depth;
 *   - ties: per-node top-k by (log q~ desc, token asc); frontier by
 *     (score desc, parent slot asc, rank-in-parent-list asc); pruning by
 *     (score desc, node id asc) with node id = (depth-1)*W + frontier rank, so
 *     ancestors always have smaller ids (the "ancestors preferred" rule of
 *     Lemma 1);
 *   - candidates with score -inf (probability zero) are never retained.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

typedef struct {
    int V, d, L, W, k, B, nseq, pos_offset, wdtype; /* wdtype 0: float32, 1: bf16 bits */
    int cand_k;                                     /* K of Algorithm 1; 0 = full vocabulary */
    double beta, temperature, rms_eps;
} orc_cfg;

int orc_num_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* ---------------------------------------------------------------- weights */

static double bf16_to_double(uint16_t b) {
    uint32_t u = (uint32_t)b << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

static double wval(const void *w, int dt, size_t i) {
    return dt == 0 ? (double)((const float *)w)[i] : bf16_to_double(((const uint16_t *)w)[i]);
}

/* sum_j w[off + j] * x[j], j < n, accumulated in fp64 in index order. */
static double wdot(const void *w, int dt, size_t off, const double *x, int n) {
    double acc = 0.0;
    if (dt == 0) {
        const float *p = (const float *)w + off;
        for (int j = 0; j < n; j++) acc += (double)p[j] * x[j];
    } else {
        const uint16_t *p = (const uint16_t *)w + off;
        for (int j = 0; j < n; j++) acc += bf16_to_double(p[j]) * x[j];
    }
    return acc;
}

/* ------------------------------------------------------ correction head g */

/* Fallback head: x = [h_p ; E[tok]] (2d), u = W_i x, a = SiLU(u), y = W_o a,
 * h_c = RMSNorm(h_p + y) = r / sqrt(mean(r^2) + eps).  W_i is [d][2d], W_o is
 * [d][d], both row-major with the output feature as the row. */
void orc_head(const orc_cfg *c, const void *Wi, const void *Wo, const void *E,
              const double *hp, int tok, double *hc) {
    const int d = c->d, dt = c->wdtype;
    double *x = (double *)malloc(sizeof(double) * 2 * (size_t)d);
    double *a = (double *)malloc(sizeof(double) * (size_t)d);
    double *r = (double *)malloc(sizeof(double) * (size_t)d);
    for (int j = 0; j < d; j++) {
        x[j] = hp[j];
        x[d + j] = wval(E, dt, (size_t)tok * d + j);
    }
#pragma omp parallel for schedule(static)
    for (int i = 0; i < d; i++) {
        double u = wdot(Wi, dt, (size_t)i * 2 * d, x, 2 * d);
        a[i] = u / (1.0 + exp(-u));
    }
#pragma omp parallel for schedule(static)
    for (int i = 0; i < d; i++) r[i] = hp[i] + wdot(Wo, dt, (size_t)i * d, a, d);
    double ss = 0.0;
    for (int i = 0; i < d; i++) ss += r[i] * r[i];
    double inv = 1.0 / sqrt(ss / d + c->rms_eps);
    for (int i = 0; i < d; i++) hc[i] = r[i] * inv;
    free(x);
    free(a);
    free(r);
}

/* ------------------------------------------- corrected child distribution */

/* z[v] = (Dlog_row[v] + E[v] . h) / T' for every token v of the vocabulary. */
void orc_child_logits(const orc_cfg *c, const void *E, const float *dlog_row,
                      const double *h, double *z) {
    const double Tp = c->temperature > 0.0 ? c->temperature : 1.0;
    const int d = c->d, dt = c->wdtype;
#pragma omp parallel for schedule(static)
    for (int v = 0; v < c->V; v++)
        z[v] = ((double)dlog_row[v] + wdot(E, dt, (size_t)v * d, h, d)) / Tp;
}

/* log q~[v] = min(z[v] - logsumexp(z), 0); returns logsumexp(z).  A row whose
 * logits are all -inf has no child with nonzero probability. */
double orc_log_softmax(const double *z, int V, double *logq) {
    double m = -INFINITY;
    for (int v = 0; v < V; v++)
        if (z[v] > m) m = z[v];
    if (m == -INFINITY) {
        for (int v = 0; v < V; v++) logq[v] = -INFINITY;
        return -INFINITY;
    }
    double s = 0.0;
    for (int v = 0; v < V; v++) s += exp(z[v] - m);
    const double lse = m + log(s);
    for (int v = 0; v < V; v++) {
        double t = z[v] - lse;
        logq[v] = t < 0.0 ? t : 0.0;
    }
    return lse;
}

/* ------------------------------------------ restricted candidate set C_d */

static int int_cmp(const void *a_, const void *b_) {
    const int a = *(const int *)a_, b = *(const int *)b_;
    return (a > b) - (a < b);
}

void orc_topk(const double *x, int n, int kk, int *idx);

/* C_d = TopK(L_d^base, K) (Algorithm 1): the cand_k tokens with the largest
 * base (drafter) logits of this position, ties by token asc, returned sorted
 * by token id. */
void orc_candidates(const orc_cfg *c, const float *dlog_row, int *cand) {
    double *x = (double *)malloc(sizeof(double) * (size_t)c->V);
    for (int v = 0; v < c->V; v++) x[v] = (double)dlog_row[v];
    orc_topk(x, c->V, c->cand_k, cand);
    qsort(cand, (size_t)c->cand_k, sizeof(int), int_cmp);
    free(x);
}

/* Corrected child distribution over the candidates only (Algorithm 1 applies
 * g to C_d): z_i = (Dlog[C_i] + E[C_i] . h) / T', log q~_i = min(z_i -
 * logsumexp_i z, 0).  Returns the log-sum-exp over C_d. */
double orc_restricted_logq(const orc_cfg *c, const void *E, const float *dlog_row,
                           const int *cand, const double *h, double *lq) {
    const double Tp = c->temperature > 0.0 ? c->temperature : 1.0;
    const int K = c->cand_k, d = c->d, dt = c->wdtype;
    double *z = (double *)malloc(sizeof(double) * (size_t)K);
    for (int i = 0; i < K; i++)
        z[i] = ((double)dlog_row[cand[i]] + wdot(E, dt, (size_t)cand[i] * d, h, d)) / Tp;
    double lse = orc_log_softmax(z, K, lq);
    free(z);
    return lse;
}

/* Corrected log-probabilities of every token (tokens outside C_d: -inf) and
 * the log-sum-exp; full vocabulary when cand_k = 0. */
static double child_logq_all(const orc_cfg *c, const void *E, const float *dlog_row, const double *h,
                             double *lq_all) {
    const int V = c->V;
    if (c->cand_k <= 0) {
        double *z = (double *)malloc(sizeof(double) * (size_t)V);
        orc_child_logits(c, E, dlog_row, h, z);
        double lse = orc_log_softmax(z, V, lq_all);
        free(z);
        return lse;
    }
    int *cand = (int *)malloc(sizeof(int) * (size_t)c->cand_k);
    double *lq = (double *)malloc(sizeof(double) * (size_t)c->cand_k);
    orc_candidates(c, dlog_row, cand);
    double lse = orc_restricted_logq(c, E, dlog_row, cand, h, lq);
    for (int v = 0; v < V; v++) lq_all[v] = -INFINITY;
    for (int i = 0; i < c->cand_k; i++) lq_all[cand[i]] = lq[i];
    free(cand);
    free(lq);
    return lse;
}

static int better(double a, int ia, double b, int ib) {
    return a > b || (a == b && ia < ib);
}

/* Indices of the kk best entries of x by (value desc, index asc), best first. */
void orc_topk(const double *x, int n, int kk, int *idx) {
    int cnt = 0;
    for (int v = 0; v < n; v++) {
        if (cnt == kk && !better(x[v], v, x[idx[kk - 1]], idx[kk - 1])) continue;
        int pos = cnt < kk ? cnt++ : kk - 1;
        while (pos > 0 && better(x[v], v, x[idx[pos - 1]], idx[pos - 1])) {
            idx[pos] = idx[pos - 1];
            pos--;
        }
        idx[pos] = v;
    }
}

/* ------------------------------------------------------------ Algorithm 1 */

typedef struct {
    double score;
    int p, j, tok;
} cand_t;

static int cand_cmp(const void *a_, const void *b_) {
    const cand_t *a = (const cand_t *)a_, *b = (const cand_t *)b_;
    if (a->score > b->score) return -1;
    if (a->score < b->score) return 1;
    if (a->p != b->p) return a->p < b->p ? -1 : 1;
    if (a->j != b->j) return a->j < b->j ? -1 : 1;
    return 0;
}

typedef struct {
    double score;
    int id;
} node_t;

static int node_cmp(const void *a_, const void *b_) {
    const node_t *a = (const node_t *)a_, *b = (const node_t *)b_;
    if (a->score > b->score) return -1;
    if (a->score < b->score) return 1;
    return a->id < b->id ? -1 : (a->id > b->id);
}

/* Children listed per node: k + 1 (one more than kept, for rank-gap checks),
 * at most the number of candidates. */
static int kx_of(const orc_cfg *c) {
    const int n = c->cand_k > 0 ? c->cand_k : c->V;
    return c->k + 1 <= n ? c->k + 1 : n;
}

/* Emission for one sequence: global top-B over the supertree (Algorithm 1,
 * final step), flattened in ascending node id, which is a topological order.
 * Output rows beyond the selected count are padding.  Returns 0, or -1 if a
 * selected node's parent was not selected (impossible when beta <= 0). */
static int prune_emit_one(const orc_cfg *c, int s, const int *st_tok, const int *st_parent,
                          const double *st_score, const int *st_count, int *o_tok, int *o_par,
                          int *o_dep, int *o_pos, double *o_score, int *o_n, uint64_t *o_mask,
                          double *prune_gap) {
    const int L = c->L, W = c->W, B = c->B, nw = (B + 63) / 64;
    const int base = s * L * W;
    node_t *nodes = (node_t *)malloc(sizeof(node_t) * (size_t)L * W + 1);
    int total = 0;
    for (int dep = 1; dep <= L; dep++)
        for (int r = 0; r < st_count[s * L + dep - 1]; r++) {
            int id = (dep - 1) * W + r;
            nodes[total].score = st_score[base + id];
            nodes[total].id = id;
            total++;
        }
    qsort(nodes, (size_t)total, sizeof(node_t), node_cmp);
    const int beff = total < B ? total : B;
    prune_gap[s] = total > beff ? nodes[beff - 1].score - nodes[beff].score : INFINITY;
    int *out_idx = (int *)malloc(sizeof(int) * (size_t)L * W);
    char *sel = (char *)calloc((size_t)L * W, 1);
    for (int i = 0; i < L * W; i++) out_idx[i] = -1;
    for (int i = 0; i < beff; i++) sel[nodes[i].id] = 1;
    int rc = 0, n = 0;
    for (int id = 0; id < L * W; id++) {
        if (!sel[id]) continue;
        out_idx[id] = n;
        const int dep = id / W + 1;
        int par = -1;
        if (dep > 1) {
            int pid = (dep - 2) * W + st_parent[base + id];
            par = out_idx[pid];
            if (par < 0) rc = -1;
        }
        const size_t o = (size_t)s * B + n;
        o_tok[o] = st_tok[base + id];
        o_par[o] = par;
        o_dep[o] = dep;
        o_pos[o] = c->pos_offset + dep;
        o_score[o] = st_score[base + id];
        uint64_t *row = o_mask + o * nw;
        memset(row, 0, sizeof(uint64_t) * nw);
        /* bit j of row n is set iff j is n itself or one of its ancestors */
        row[n / 64] |= 1ull << (n % 64);
        int a = par;
        while (a >= 0) {
            row[a / 64] |= 1ull << (a % 64);
            a = o_par[(size_t)s * B + a];
        }
        n++;
    }
    for (int i = n; i < B; i++) {
        const size_t o = (size_t)s * B + i;
        o_tok[o] = -1;
        o_par[o] = -2;
        o_dep[o] = 0;
        o_pos[o] = -1;
        o_score[o] = -INFINITY;
        memset(o_mask + o * nw, 0, sizeof(uint64_t) * nw);
    }
    o_n[s] = n;
    free(nodes);
    free(out_idx);
    free(sel);
    return rc;
}

/* Top-B pruning + emission of every sequence of a given supertree. */
int orc_prune_emit(const orc_cfg *c, const int *st_tok, const int *st_parent,
                   const double *st_score, const int *st_count, int *o_tok, int *o_par,
                   int *o_dep, int *o_pos, double *o_score, int *o_n, uint64_t *o_mask,
                   double *prune_gap) {
    int rc = 0;
    for (int s = 0; s < c->nseq; s++)
        if (prune_emit_one(c, s, st_tok, st_parent, st_score, st_count, o_tok, o_par, o_dep,
                           o_pos, o_score, o_n, o_mask, prune_gap))
            rc = -1;
    return rc;
}

/* Algorithm 1 for every sequence, followed by pruning and emission.
 * Arrays (all caller-allocated, row-major):
 *   Dlog [nseq][L][V] float, h0 [nseq][d] float;
 *   supertree st_tok / st_parent (slot in the previous depth, -1 = root) /
 *     st_score [nseq][L][W], st_count [nseq][L];
 *   per expanded node p of depth d-1 (index [s][d-1][p]): nd_lse, and its
 *     kx = min(k+1, V) best children nd_tok / nd_logq [..][kx];
 *   fr_score [nseq][L][W+1]: the W+1 best candidate scores at each depth;
 *   emitted tree o_* [nseq][B], o_mask [nseq][B][ceil(B/64)], o_n [nseq],
 *   prune_gap [nseq] (score gap at the budget cut, +inf if nothing was cut).
 * Returns 0 on success. */
int orc_build_tree(const orc_cfg *c, const void *Wi, const void *Wo, const void *E,
                   const float *Dlog, const float *h0, int *st_tok, int *st_parent,
                   double *st_score, int *st_count, double *nd_lse, int *nd_tok,
                   double *nd_logq, double *fr_score, int *o_tok, int *o_par, int *o_dep,
                   int *o_pos, double *o_score, int *o_n, uint64_t *o_mask, double *prune_gap) {
    const int V = c->V, d = c->d, L = c->L, W = c->W, k = c->k, kx = kx_of(c);
    /* entries scored per node: every token, or the candidate set C_d
     * (ent[i] = token of entry i, ascending) */
    const int nent = c->cand_k > 0 ? c->cand_k : V;
    double *hs = (double *)malloc(sizeof(double) * (size_t)W * d);
    double *hn = (double *)malloc(sizeof(double) * (size_t)W * d);
    double *z = (double *)malloc(sizeof(double) * (size_t)V);
    double *logq = (double *)malloc(sizeof(double) * (size_t)V);
    int *ent = (int *)malloc(sizeof(int) * (size_t)nent);
    int *idx = (int *)malloc(sizeof(int) * (size_t)kx);
    for (int i = 0; i < nent; i++) ent[i] = i;
    cand_t *cand = (cand_t *)malloc(sizeof(cand_t) * (size_t)W * k + 1);
    double pscore[1024], nscore[1024];
    int rc = 0;
    for (int s = 0; s < c->nseq; s++) {
        /* S_0 = {root}, r(root) = h_0, s_beta(root) = 0 */
        for (int j = 0; j < d; j++) hs[j] = (double)h0[(size_t)s * d + j];
        pscore[0] = 0.0;
        int pcount = 1;
        for (int dep = 1; dep <= L; dep++) {
            const float *row = Dlog + ((size_t)s * L + dep - 1) * V;
            const size_t nb = ((size_t)s * L + dep - 1) * W;
            if (c->cand_k > 0) orc_candidates(c, row, ent); /* C_d = TopK(L_d^base, K) */
            int ncand = 0;
            for (int p = 0; p < W; p++) {
                nd_lse[nb + p] = -INFINITY;
                for (int j = 0; j < kx; j++) {
                    nd_tok[(nb + p) * kx + j] = -1;
                    nd_logq[(nb + p) * kx + j] = -INFINITY;
                }
            }
            /* score every child of every retained prefix in S_{d-1} */
            for (int p = 0; p < pcount; p++) {
                if (c->cand_k > 0) {
                    nd_lse[nb + p] = orc_restricted_logq(c, E, row, ent, hs + (size_t)p * d, logq);
                } else {
                    orc_child_logits(c, E, row, hs + (size_t)p * d, z);
                    nd_lse[nb + p] = orc_log_softmax(z, V, logq);
                }
                /* entries are in token order, so index ties are token ties */
                orc_topk(logq, nent, kx, idx);
                for (int j = 0; j < kx; j++) {
                    nd_tok[(nb + p) * kx + j] = ent[idx[j]];
                    nd_logq[(nb + p) * kx + j] = logq[idx[j]];
                }
                for (int j = 0; j < k; j++) {
                    cand[ncand].score = pscore[p] + logq[idx[j]] + c->beta; /* Eq. 5 */
                    cand[ncand].p = p;
                    cand[ncand].j = j;
                    cand[ncand].tok = ent[idx[j]];
                    ncand++;
                }
            }
            qsort(cand, (size_t)ncand, sizeof(cand_t), cand_cmp);
            int nvalid = 0;
            while (nvalid < ncand && cand[nvalid].score > -INFINITY) nvalid++;
            const int cnt = nvalid < W ? nvalid : W; /* global top-W -> S_d */
            for (int r = 0; r <= W; r++)
                fr_score[((size_t)s * L + dep - 1) * (W + 1) + r] =
                    r < nvalid ? cand[r].score : -INFINITY;
            const size_t sb = ((size_t)s * L + dep - 1) * W;
            for (int r = 0; r < W; r++) {
                st_tok[sb + r] = r < cnt ? cand[r].tok : -1;
                st_parent[sb + r] = r < cnt ? cand[r].p : -1;
                st_score[sb + r] = r < cnt ? cand[r].score : -INFINITY;
            }
            st_count[s * L + dep - 1] = cnt;
            /* carry the correction states of the retained children */
            if (dep < L)
                for (int r = 0; r < cnt; r++)
                    orc_head(c, Wi, Wo, E, hs + (size_t)cand[r].p * d, cand[r].tok,
                             hn + (size_t)r * d);
            for (int r = 0; r < cnt; r++) nscore[r] = cand[r].score;
            memcpy(pscore, nscore, sizeof(double) * (size_t)cnt);
            double *t = hs;
            hs = hn;
            hn = t;
            pcount = cnt;
        }
    }
    if (orc_prune_emit(c, st_tok, st_parent, st_score, st_count, o_tok, o_par, o_dep, o_pos,
                       o_score, o_n, o_mask, prune_gap))
        rc = -1;
    free(hs);
    free(hn);
    free(z);
    free(logq);
    free(ent);
    free(idx);
    free(cand);
    return rc;
}

/* ----------------------------------------------- best-first heap (Lemma 1) */

/* Best-first selection over a materialised supertree of sequence s: a max-heap
 * seeded with the root's children; each pop emits the best prefix and pushes
 * its materialised children; stops after min(B, |S|) pops.  Writes the popped
 * node ids in pop order and returns their count. */
int orc_heap_select(const orc_cfg *c, const int *st_parent, const double *st_score,
                    const int *st_count, int s, int *popped) {
    const int L = c->L, W = c->W;
    const int base = s * L * W;
    int total = 0;
    for (int dep = 1; dep <= L; dep++) total += st_count[s * L + dep - 1];
    const int beff = total < c->B ? total : c->B;
    node_t *heap = (node_t *)malloc(sizeof(node_t) * ((size_t)L * W + 1));
    int hn = 0, np = 0;
#define HBETTER(a, b) ((a).score > (b).score || ((a).score == (b).score && (a).id < (b).id))
#define HPUSH(nd)                                                  \
    do {                                                           \
        int i_ = hn++;                                             \
        heap[i_] = (nd);                                           \
        while (i_ > 0 && HBETTER(heap[i_], heap[(i_ - 1) / 2])) {  \
            node_t t_ = heap[i_];                                  \
            heap[i_] = heap[(i_ - 1) / 2];                         \
            heap[(i_ - 1) / 2] = t_;                               \
            i_ = (i_ - 1) / 2;                                     \
        }                                                          \
    } while (0)
    for (int r = 0; r < st_count[s * L]; r++) {
        node_t nd = {st_score[base + r], r};
        HPUSH(nd);
    }
    while (np < beff && hn > 0) {
        node_t top = heap[0];
        heap[0] = heap[--hn];
        int i = 0;
        for (;;) {
            int l = 2 * i + 1, rr = l + 1, b = i;
            if (l < hn && HBETTER(heap[l], heap[b])) b = l;
            if (rr < hn && HBETTER(heap[rr], heap[b])) b = rr;
            if (b == i) break;
            node_t t = heap[i];
            heap[i] = heap[b];
            heap[b] = t;
            i = b;
        }
        popped[np++] = top.id;
        const int dep = top.id / W + 1, slot = top.id % W;
        if (dep < L)
            for (int r = 0; r < st_count[s * L + dep]; r++)
                if (st_parent[base + dep * W + r] == slot) {
                    node_t ch = {st_score[base + dep * W + r], dep * W + r};
                    HPUSH(ch);
                }
    }
#undef HPUSH
#undef HBETTER
    free(heap);
    return np;
}

/* ----------------------------------------------- teacher-forced path tools */

/* State r(u) of the prefix u = path[0..len) of sequence (Dlog_seq, h0_seq),
 * obtained by running the correction head from the root along the path. */
void orc_path_state(const orc_cfg *c, const void *Wi, const void *Wo, const void *E,
                    const float *h0_seq, const int *path, int len, double *h_out) {
    const int d = c->d;
    double *h = (double *)malloc(sizeof(double) * (size_t)d);
    double *t = (double *)malloc(sizeof(double) * (size_t)d);
    for (int j = 0; j < d; j++) h[j] = (double)h0_seq[j];
    for (int i = 0; i < len; i++) {
        orc_head(c, Wi, Wo, E, h, path[i], t);
        memcpy(h, t, sizeof(double) * (size_t)d);
    }
    memcpy(h_out, h, sizeof(double) * (size_t)d);
    free(h);
    free(t);
}

/* Children of the prefix path[0..len): its corrected log-probabilities over
 * the whole vocabulary (logq_all, may be NULL), their log-sum-exp, and the kk
 * best children by (log q~ desc, token asc). */
double orc_node_children(const orc_cfg *c, const void *Wi, const void *Wo, const void *E,
                         const float *Dlog_seq, const float *h0_seq, const int *path, int len,
                         int kk, int *tok_out, double *logq_out, double *logq_all) {
    const int V = c->V, d = c->d;
    double *h = (double *)malloc(sizeof(double) * (size_t)d);
    double *lq = logq_all ? logq_all : (double *)malloc(sizeof(double) * (size_t)V);
    orc_path_state(c, Wi, Wo, E, h0_seq, path, len, h);
    const float *row = Dlog_seq + (size_t)len * V;
    double lse = child_logq_all(c, E, row, h, lq);
    if (kk > 0) {
        if (c->cand_k > 0) {
            /* the kk best candidates (kk <= cand_k), ties by token asc */
            int *cand = (int *)malloc(sizeof(int) * (size_t)c->cand_k);
            double *lc = (double *)malloc(sizeof(double) * (size_t)c->cand_k);
            orc_candidates(c, row, cand);
            for (int i = 0; i < c->cand_k; i++) lc[i] = lq[cand[i]];
            orc_topk(lc, c->cand_k, kk, tok_out);
            for (int j = 0; j < kk; j++) {
                logq_out[j] = lc[tok_out[j]];
                tok_out[j] = cand[tok_out[j]];
            }
            free(cand);
            free(lc);
        } else {
            orc_topk(lq, V, kk, tok_out);
            for (int j = 0; j < kk; j++) logq_out[j] = lq[tok_out[j]];
        }
    }
    free(h);
    if (!logq_all) free(lq);
    return lse;
}

/* Eq. 5 along a path: scores[i] = sum_{i' <= i} log q~(path[i']) + beta (i+1). */
void orc_path_scores(const orc_cfg *c, const void *Wi, const void *Wo, const void *E,
                     const float *Dlog_seq, const float *h0_seq, const int *path, int len,
                     double *scores) {
    const int V = c->V, d = c->d;
    double *h = (double *)malloc(sizeof(double) * (size_t)d);
    double *t = (double *)malloc(sizeof(double) * (size_t)d);
    double *lq = (double *)malloc(sizeof(double) * (size_t)V);
    for (int j = 0; j < d; j++) h[j] = (double)h0_seq[j];
    double s = 0.0;
    for (int i = 0; i < len; i++) {
        child_logq_all(c, E, Dlog_seq + (size_t)i * V, h, lq);
        s += lq[path[i]] + c->beta;
        scores[i] = s;
        if (i + 1 < len) {
            orc_head(c, Wi, Wo, E, h, path[i], t);
            memcpy(h, t, sizeof(double) * (size_t)d);
        }
    }
    free(h);
    free(t);
    free(lq);
}

/* ------------------------------------------- heap-based constructions */

/* Emission of a tree built by best-first popping (rows in pop order, which is
 * a topological order: a node is popped after its parent).  Row i holds
 * token tok[i], parent row par[i] (-1: the root), depth dep[i] and score
 * sc[i]; mask rows by the ancestor walk; rows n..B-1 are padding. */
static void emit_pop_order(const orc_cfg *c, int s, int n, const int *tok, const int *par, const int *dep,
                           const double *sc, int *o_tok, int *o_par, int *o_dep, int *o_pos, double *o_score,
                           int *o_n, uint64_t *o_mask) {
    const int B = c->B, nw = (B + 63) / 64;
    for (int i = 0; i < B; i++) {
        const size_t o = (size_t)s * B + i;
        uint64_t *row = o_mask + o * nw;
        memset(row, 0, sizeof(uint64_t) * nw);
        if (i < n) {
            o_tok[o] = tok[i];
            o_par[o] = par[i];
            o_dep[o] = dep[i];
            o_pos[o] = c->pos_offset + dep[i];
            o_score[o] = sc[i];
            for (int a = i; a >= 0; a = par[a]) row[a / 64] |= 1ull << (a % 64);
        } else {
            o_tok[o] = -1;
            o_par[o] = -2;
            o_dep[o] = 0;
            o_pos[o] = -1;
            o_score[o] = -INFINITY;
        }
    }
    o_n[s] = n;
}

/* Sorted child list of a distribution: the m = min(B, entries) best
 * (log q~ desc, token asc) tokens and their log q~.  lq_all holds log q~ of
 * every token (-inf outside C_d when the candidate set is restricted). */
static int child_list(const orc_cfg *c, const double *lq_all, int *ltok, double *llq) {
    const int nent = c->cand_k > 0 ? c->cand_k : c->V;
    const int m = c->B < nent ? c->B : nent;
    orc_topk(lq_all, c->V, m, ltok);
    for (int j = 0; j < m; j++) llq[j] = lq_all[ltok[j]];
    return m;
}

/* One best-first step over the popped nodes (and the root, index -1): every
 * node p with depth < L offers its best child not yet taken, child rank
 * next[p] of its sorted list, scored s_p + log q~ + beta (Eq. 5).  Returns
 * the node whose offer is best by (score desc, node asc; the root first), or
 * -2 if no finite offer remains.  lists: row p+1 of ltok/llq/llen. */
static int best_offer(const orc_cfg *c, int n, const int *dep, const double *sc, const int *next,
                      const int *llen, const double *llq, int lstride, double *best_score) {
    int best = -2;
    double bs = -INFINITY;
    for (int p = -1; p < n; p++) {
        const int dp = p < 0 ? 0 : dep[p];
        if (dp >= c->L || next[p + 1] >= llen[p + 1]) continue;
        const double v = (p < 0 ? 0.0 : sc[p]) + llq[(size_t)(p + 1) * lstride + next[p + 1]] + c->beta;
        if (v == -INFINITY) continue;
        if (best == -2 || v > bs) { /* p ascends, so ties keep the earlier node */
            best = p;
            bs = v;
        }
    }
    *best_score = bs;
    return best;
}

/* Domino-chain + DDTree (Sec. 5.2, Table 2): causal correction along ONE draft
 * chain, then DDTree (Sec. 3.3) over the chain-conditioned distributions.
 * Per sequence:
 *   1. the chain: from r_0, at each depth d = 1..L the corrected distribution
 *      q~_d(. | y_<d) of the chain prefix (over V, or over C_d when cand_k > 0),
 *      its argmax y_d (log q~ desc, token asc), and, for d < L, the state
 *      r(y_1..y_d) = g(r(y_<d), y_d);
 *   2. DDTree: the chain's distributions are used as position-wise marginals
 *      shared by every node of a depth; best-first search over prefixes
 *      scored s = sum_i log q~_i(u_i) + beta d (beta = 0: DDTree's mass
 *      objective), each pop taking the best offer (next child in
 *      sorted order of a popped node, DDTree's "next sibling / first child"
 *      pushes), until B nodes are popped.
 * Emitted in pop order; chain_tok / chain_lse [nseq][L] receive the chain and
 * the log-sum-exp of each of its distributions. */
int orc_chain_ddtree(const orc_cfg *c, const void *Wi, const void *Wo, const void *E, const float *Dlog,
                     const float *h0, int *chain_tok, double *chain_lse, int *o_tok, int *o_par, int *o_dep,
                     int *o_pos, double *o_score, int *o_n, uint64_t *o_mask) {
    const int V = c->V, d = c->d, L = c->L, B = c->B;
    double *h = (double *)malloc(sizeof(double) * (size_t)d);
    double *t = (double *)malloc(sizeof(double) * (size_t)d);
    double *lq = (double *)malloc(sizeof(double) * (size_t)V);
    int *ltok = (int *)malloc(sizeof(int) * (size_t)L * B);     /* per depth */
    double *llq = (double *)malloc(sizeof(double) * (size_t)L * B);
    int *llen = (int *)malloc(sizeof(int) * (size_t)L);
    int *ptok = (int *)malloc(sizeof(int) * (size_t)B), *ppar = (int *)malloc(sizeof(int) * (size_t)B);
    int *pdep = (int *)malloc(sizeof(int) * (size_t)B), *next = (int *)malloc(sizeof(int) * (size_t)(B + 1));
    int *olen = (int *)malloc(sizeof(int) * (size_t)(B + 1));
    double *psc = (double *)malloc(sizeof(double) * (size_t)B);
    double *olq = (double *)malloc(sizeof(double) * (size_t)(B + 1) * B); /* offers per node, by its depth */
    for (int s = 0; s < c->nseq; s++) {
        /* 1. the chain */
        for (int j = 0; j < d; j++) h[j] = (double)h0[(size_t)s * d + j];
        for (int dep = 1; dep <= L; dep++) {
            const float *drow = Dlog + ((size_t)s * L + dep - 1) * V; /* position dep-1 */
            chain_lse[(size_t)s * L + dep - 1] = child_logq_all(c, E, drow, h, lq);
            llen[dep - 1] = child_list(c, lq, ltok + (size_t)(dep - 1) * B, llq + (size_t)(dep - 1) * B);
            const int y = ltok[(size_t)(dep - 1) * B];
            chain_tok[(size_t)s * L + dep - 1] = y;
            if (dep < L) {
                orc_head(c, Wi, Wo, E, h, y, t);
                memcpy(h, t, sizeof(double) * (size_t)d);
            }
        }
        /* 2. DDTree over the chain-conditioned marginals */
        int n = 0;
        next[0] = 0;
        olen[0] = llen[0];
        memcpy(olq, llq, sizeof(double) * (size_t)B);
        while (n < B) {
            double v;
            const int p = best_offer(c, n, pdep, psc, next, olen, olq, B, &v);
            if (p == -2) break;
            const int dep = p < 0 ? 1 : pdep[p] + 1;
            ptok[n] = ltok[(size_t)(dep - 1) * B + next[p + 1]];
            ppar[n] = p;
            pdep[n] = dep;
            psc[n] = v;
            next[p + 1]++;
            next[n + 1] = 0;
            olen[n + 1] = dep < L ? llen[dep] : 0;
            if (dep < L) memcpy(olq + (size_t)(n + 1) * B, llq + (size_t)dep * B, sizeof(double) * (size_t)B);
            n++;
        }
        emit_pop_order(c, s, n, ptok, ppar, pdep, psc, o_tok, o_par, o_dep, o_pos, o_score, o_n, o_mask);
    }
    free(h); free(t); free(lq); free(ltok); free(llq); free(llen);
    free(ptok); free(ppar); free(pdep); free(next); free(olen); free(psc); free(olq);
    return 0;
}

/* Sequential correction with heap (Sec. 4.1, Table 2): exact node-wise
 * best-first search under the corrected scores.  The root's children are
 * scored at r_0; each pop takes the best offer among the popped nodes (each
 * offers its best child not yet taken, by its OWN corrected distribution),
 * and the popped node, if above depth L, is then corrected: its state
 * r(u_1..u_d) = g(r(u_<d), u_d) and its children's distribution
 * q~_{d+1}(. | u_1..u_d) are computed before the next pop.  B pops; emitted in
 * pop order.  expansions[s] receives the number of correction-head
 * evaluations of children (the root included). */
int orc_seq_heap(const orc_cfg *c, const void *Wi, const void *Wo, const void *E, const float *Dlog,
                 const float *h0, int *o_tok, int *o_par, int *o_dep, int *o_pos, double *o_score, int *o_n,
                 uint64_t *o_mask, int *expansions) {
    const int V = c->V, d = c->d, L = c->L, B = c->B;
    double *hs = (double *)malloc(sizeof(double) * (size_t)(B + 1) * d); /* row p+1: state of node p */
    double *lq = (double *)malloc(sizeof(double) * (size_t)V);
    int *ltok = (int *)malloc(sizeof(int) * (size_t)(B + 1) * B);
    double *llq = (double *)malloc(sizeof(double) * (size_t)(B + 1) * B);
    int *llen = (int *)malloc(sizeof(int) * (size_t)(B + 1));
    int *next = (int *)malloc(sizeof(int) * (size_t)(B + 1));
    int *ptok = (int *)malloc(sizeof(int) * (size_t)B), *ppar = (int *)malloc(sizeof(int) * (size_t)B);
    int *pdep = (int *)malloc(sizeof(int) * (size_t)B);
    double *psc = (double *)malloc(sizeof(double) * (size_t)B);
    for (int s = 0; s < c->nseq; s++) {
        const float *dl = Dlog + (size_t)s * L * V;
        for (int j = 0; j < d; j++) hs[j] = (double)h0[(size_t)s * d + j];
        child_logq_all(c, E, dl, hs, lq);
        llen[0] = child_list(c, lq, ltok, llq);
        next[0] = 0;
        int n = 0, nexp = 1;
        while (n < B) {
            double v;
            const int p = best_offer(c, n, pdep, psc, next, llen, llq, B, &v);
            if (p == -2) break;
            const int dep = p < 0 ? 1 : pdep[p] + 1;
            const int tk = ltok[(size_t)(p + 1) * B + next[p + 1]];
            ptok[n] = tk;
            ppar[n] = p;
            pdep[n] = dep;
            psc[n] = v;
            next[p + 1]++;
            next[n + 1] = 0;
            llen[n + 1] = 0;
            if (dep < L) { /* correct the new prefix: its state, then its children */
                double *hn = hs + (size_t)(n + 1) * d;
                orc_head(c, Wi, Wo, E, hs + (size_t)(p + 1) * d, tk, hn);
                child_logq_all(c, E, dl + (size_t)dep * V, hn, lq);
                llen[n + 1] = child_list(c, lq, ltok + (size_t)(n + 1) * B, llq + (size_t)(n + 1) * B);
                nexp++;
            }
            n++;
        }
        expansions[s] = nexp;
        emit_pop_order(c, s, n, ptok, ppar, pdep, psc, o_tok, o_par, o_dep, o_pos, o_score, o_n, o_mask);
    }
    free(hs); free(lq); free(ltok); free(llq); free(llen); free(next);
    free(ptok); free(ppar); free(pdep); free(psc);
    return 0;
}
