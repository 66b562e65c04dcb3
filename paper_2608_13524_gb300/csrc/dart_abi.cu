// C ABI of the DARTree construction path: argument validation, workspace,
// TMA tensor maps, per-depth orchestration of the kernels (Algorithm 1),
// pruning/emission, CUDA-graph caching of whole rounds, the host-buffer
// variant and the test hooks.  See include/dart.h for the contract.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <new>
#include <vector>

#include "../../include/dart.h"
#include "dart_device.cuh"
#include "dart_kernels.h"

dart::EncodeTiledFn dart::tensor_map_encoder() {
    static EncodeTiledFn fn = nullptr;
    if (!fn) {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    }
    return fn;
}

using namespace dart;

namespace {

constexpr int kVersion = 2;
constexpr int kMaxW = 64, kMaxK = 64, kMaxWK = 4096, kMaxSuper = 1024, kMaxB = 1024;
constexpr int kMaxD = 16384;
constexpr int kMaxCandK = 1024;  // candidate-set size K of the restricted scoring
constexpr int kMaxV = (1 << 24) - 1;
constexpr int kMaxProfilePairs = 8192;
constexpr size_t kMaxGraphs = 8;  // cached round graphs per handle (least recently used evicted)

EncodeTiledFn encode_fn() { return tensor_map_encoder(); }

// 2-D bf16 tensor [rows][inner] (row pitch `pitch` elements, default inner)
// with a (64 x box_rows) box and 128-byte swizzle.
bool encode_bf16_2d(CUtensorMap* m, const void* base, uint64_t inner, uint64_t rows, uint32_t box_rows,
                    uint64_t pitch = 0) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {inner, rows};
    cuuint64_t strides[1] = {(pitch ? pitch : inner) * 2};
    cuuint32_t box[2] = {static_cast<cuuint32_t>(kBlockK), box_rows};
    cuuint32_t estr[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
bool aligned4(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 3u) == 0; }

int ng_index(int NG) { return NG == 16 ? 0 : (NG == 32 ? 1 : (NG == 64 ? 2 : 3)); }

struct DepthPlan {
    int N, P, NG, G, nV, stages, smem;  // LM-head scoring
    int l2pf;                            // LM-head: E tiles per CTA prefetched into L2 before its wait
    int epf;                             // of those and the stages, how many the previous depth prefetches early
    int bound;                           // seed rows per sequence of the seed pass before this depth's LM-head (0: none)
    int nlist, klist;                    // sorted key lists per node and their length (merge input)
    int cand_ds;                         // candidate scoring: d slices per candidate group
    int f32_ds;                          // fp32 LM-head: blocks per vocabulary range (d slices)
    int Nc, Pn;                          // children (head update) at this depth
    int split;                           // g1 = W_i[:, 0:d] . h over the N parents; E half from the Q table
    int side;                            // split: g1 runs on the side stream beside merge + select
    GemmArgs g1, g2;                     // head GEMMs (depth < L)
    int g1_smem, g2_smem;
};

// Round graph cache key: the construction (kind) and the pointer set.
enum RoundKind { kRoundDartree = 0, kRoundChainDdtree = 1, kRoundSeqHeap = 2 };

struct GraphEntry {
    const void* key[10];
    cudaGraphExec_t exec;
    unsigned long long last_use;
};

}  // namespace

struct dart_handle {
    dart_config cfg;
    int wdtype;
    const void *Wi, *Wo, *E;
    int dev, num_sms, smem_optin;
    long long l2_bytes;   // L2 cache size (plans of the early E prefetch)
    std::vector<int> caps;
    std::vector<DepthPlan> plans;
    int next_depth;  // 1..L+1 (L+1 = all depths expanded)
    int cur;         // which state buffer holds the current frontier
    int last_rows;
    // workspace
    float* hbuf[2];
    __nv_bfloat16 *HL, *XL, *AL;
    float *X32, *A32;
    float* part;
    float2* part_ms;
    uint64_t* part_key;
    float *node_logq, *node_lse;
    int* node_tok;
    int *tree_tok, *tree_parent, *tree_count;
    float* tree_score;
    int *child_prow, *child_tok, *seq_ticket, *status;
    uint64_t* gthr;  // [L][kNPadMax] cross-CTA top-k bounds of every depth, zeroed per round
    float* bound_y;     // [kNPadMax][kBoundR] seed scores less their error bounds (topk_bound)
    int* cand_tok;   // [nseq][L][cand_k] candidate sets C_d (cand_k > 0)
    float* cand_scratch;  // candidate scoring partial dot products
    int* cand_ticket;     // [nseq][ceil(cand_k/8)]
    uint64_t* cand_part;  // [nseq * L][slices][cand_k] per-slice top keys of the candidate selection
    int* cand_rticket;    // [nseq * L] slices finished per row
    float* Qtab;          // [V][d] fp32: Q[t] = W_i[:, d:2d] . E[t] (split first head layer), or null
    // copies of the streamed weights as 128 x 64 tiles of contiguous 16 KB
    // (launch_retile), or null: E (weights_tiled), W_i and W_o (head_weights_tiled)
    bool tiled, wtiled;
    __nv_bfloat16* Et;    // E [V][d]
    __nv_bfloat16* Wit;   // W_i[:, 0:Kwi], Kwi = d with the split first layer, else 2d
    __nv_bfloat16* Wot;   // W_o
    int Kwi;
    // best-first constructions (dart_config.variants): the one-node-per-
    // sequence plans (W = k = 1) of the chain and of the sequential search
    dart_config ccfg;
    std::vector<int> ccaps;
    std::vector<DepthPlan> cplans;
    int Bp;                // children kept per distribution: min(B, V)
    int ddt_S, sh_S;       // top-K slices per row (chain rows, popped-prefix rows)
    // Domino-chain + DDTree
    float* zrows;          // [nseq][L][V] the chain's scaled logits
    float* chain_lse;      // [nseq][L]
    int* ddt_tok;          // [nseq][L][Bp]
    float* ddt_z;
    uint64_t* ddt_part;    // [nseq * L][topk_S][Bp]
    int* ddt_ticket;       // [nseq * L]
    // sequential correction with heap (slot 0 = the root, p + 1 = node p)
    float* sh_tab;         // [nseq][B+1][d]
    int* sh_ltok;          // [nseq][B+1][Bp]
    float* sh_lz;
    float* sh_llse;        // [nseq][B+1]
    int *sh_next, *sh_npop, *sh_dlog_row;
    float* sh_offer;
    float* sh_zrow;        // [nseq][V]
    uint64_t* sh_part;     // [nseq][topk_S][Bp]
    int* sh_ticket;        // [nseq]
    int last_kind;         // construction of the most recent round (RoundKind)
    // fused small-problem round (dart_config.fused_round): one cooperative
    // kernel of fused_G blocks, each scoring at most fused_R vocabulary rows
    bool fused;
    bool fused_cluster;    // one cluster per sequence (else one cooperative grid)
    int fused_nm, fused_G, fused_R;
    bool fused_ecache, fused_mstage;
    int fused_stage;       // cluster form: bytes per E stage
    bool fused_wres;       // cluster form: head weights resident in shared memory
    size_t fused_smem;
    float *f_rbuf, *f_abuf, *f_ssqp;
    float2* f_pms;
    uint64_t* f_pkey;
    unsigned* f_bar;       // grid barrier: arrivals, generation
    int* f_abort;
    bool f_dirty;          // the barrier probe left the barrier mid-way (until dart_status_sync)
    std::vector<void*> allocs;
    CUtensorMap tmE, tmWi, tmWo, tmH[4], tmX[3], tmA[3];
    CUtensorMap tmWiR, tmEB;  // Q table: A = W_i[:, d:2d] (128-row box), B = E rows as 64-node groups
    // host-buffer staging
    float *st_dlog, *st_anchor;
    dart_tree_out st_out;
    bool staged;
    // side stream of the split first head layer (fork after the LM-head,
    // join before gather_silu)
    cudaStream_t side;
    cudaEvent_t ev_fork, ev_join;
    // graphs
    cudaStream_t cap_stream;
    std::vector<GraphEntry> graphs;
    unsigned long long graph_clock;
    // profiling
    bool profiling;
    std::vector<cudaEvent_t> ev;
    std::vector<int> ev_kind;
    int ev_used;
};

namespace {

int cuda_err(cudaError_t e) { return e == cudaSuccess ? DART_OK : DART_ERR_CUDA; }

template <typename T>
int dalloc(dart_handle* h, T** p, size_t count) {
    void* q = nullptr;
    if (count == 0) count = 1;
    if (cudaMalloc(&q, count * sizeof(T)) != cudaSuccess) return DART_ERR_NOMEM;
    h->allocs.push_back(q);
    *p = static_cast<T*>(q);
    return DART_OK;
}

int validate_cfg(const dart_config* c) {
    if (!c) return DART_ERR_INVALID;
    if (c->V < 1 || c->V > kMaxV) return DART_ERR_INVALID;
    if (c->d < 64 || c->d > kMaxD || c->d % 64) return DART_ERR_INVALID;
    if (c->L < 1 || c->W < 1 || c->W > kMaxW || c->L * c->W > kMaxSuper) return DART_ERR_INVALID;
    if (c->k < 1 || c->k > kMaxK || c->k > c->V || c->W * c->k > kMaxWK) return DART_ERR_INVALID;
    if (c->B < 1 || c->B > kMaxB) return DART_ERR_INVALID;
    if (c->nseq < 1 || c->nseq * c->W > kNPadMax) return DART_ERR_INVALID;
    if (!(c->beta <= 0.0f) || !std::isfinite(c->beta)) return DART_ERR_INVALID;  // Lemma 1 needs beta <= 0
    if (!(c->temperature >= 0.0f) || !std::isfinite(c->temperature)) return DART_ERR_INVALID;
    if (!(c->rms_eps > 0.0f) || !std::isfinite(c->rms_eps)) return DART_ERR_INVALID;
    if (c->cand_k != 0 && (c->cand_k < c->k || c->cand_k > c->V || c->cand_k > kMaxCandK)) return DART_ERR_INVALID;
    for (int sw : {c->head_split, c->head_split_stream, c->weights_tiled, c->head_weights_tiled, c->fused_round,
                   c->topk_bound})
        if (sw != DART_AUTO && sw != DART_ON && sw != DART_OFF) return DART_ERR_INVALID;
    if (c->lmhead_ctas_per_sm < 0 || c->lmhead_ctas_per_sm > 2) return DART_ERR_INVALID;
    if (c->variants & ~(DART_VARIANT_CHAIN_DDTREE | DART_VARIANT_SEQ_HEAP)) return DART_ERR_INVALID;
    return DART_OK;
}

// Node group of the head GEMMs (up to 64) and of the fp32 LM-head kernel; the
// tensor-core LM-head kernel's plan comes from plan_lmhead_tc (groups of up
// to 128 nodes: one MMA of N = 256 covers the hi and lo products of 128).
int pick_ng_gemm(int N) { return N <= 16 ? 16 : (N <= 32 ? 32 : 64); }
int pick_ng_f32(int N) { return N <= 16 ? 16 : 32; }

// Split-K GEMM plan: M = d output features, K reduction, Nc nodes.
GemmArgs gemm_plan(const dart_handle* h, int K, int Nc, int lo_kb_end, bool tc) {
    GemmArgs g;
    std::memset(&g, 0, sizeof g);
    const int d = h->cfg.d;
    g.M = d;
    g.K = K;
    g.N = Nc;
    g.KB = K / kBlockK;
    g.lo_kb_end = lo_kb_end;
    g.bhalf = kNPadMax;
    if (tc) {
        g.NG = pick_ng_gemm(Nc);
        g.G = (Nc + g.NG - 1) / g.NG;
        g.MT = (d + kTileM - 1) / kTileM;
        g.S = std::max(1, std::min(g.KB, h->num_sms / (g.MT * g.G)));
    } else {
        g.NG = 16;
        g.G = (Nc + 15) / 16;
        g.MT = (d + 63) / 64;
        g.S = std::max(1, std::min(K / 32, (2 * h->num_sms) / (g.MT * g.G)));
    }
    return g;
}

constexpr long long kL2PrefetchBytes = 64ll << 20;  // about half of the 126 MB L2
// Starting bound of the LM-head's top-k filters (topk_bound): at most this
// many seed rows per sequence (2k rounded up to 64; scratch per node).
constexpr int kBoundR = 2 * kMaxK;
constexpr long long kL2KeepBytes = 72ll << 20;      // head weights kept in L2 across depths, at most

int tc_stages(int smem_optin, int stage_bytes, int fixed) {
    int s = (smem_optin - fixed) / stage_bytes;
    return std::min(16, s);
}

// Launch plans of every depth for configuration c (the handle's, or the
// one-node-per-sequence configuration of the best-first constructions).
// Whether dart_build_tree runs as one cooperative kernel (fused_round): fp32
// weights, full-vocabulary scoring, at most 32 nodes per depth, and the
// kernel's shared memory (node states, per-block score keys, selection
// buffers) within the device limit; one block per SM, at most 160.
int plan_fused_round(dart_handle* h) {
    const dart_config& c = h->cfg;
    h->fused = false;
    if (c.fused_round == DART_OFF) return DART_OK;
    int nmax = 0, pmax = 0;
    for (int dep = 1; dep <= c.L; dep++) {
        nmax = std::max(nmax, c.nseq * h->caps[dep - 1]);
        pmax = std::max(pmax, h->caps[dep - 1]);
    }
    const bool base_ok = h->wdtype == DART_F32 && c.cand_k == 0 && c.W <= 32 && c.L <= kRoundMaxL &&
                         c.L * c.W <= 256 && c.k <= 32 && c.d <= 1024;
    // the kernel's static shared memory (prune / emit and selection scratch) is below 32 KB
    const size_t avail = static_cast<size_t>(h->smem_optin) - 32 * 1024;
    {
        // one cluster per sequence: where a block's share of E (re-read at
        // every depth) is at most 512 KB and the sequence's states and slice
        // keys fit in shared memory
        const int pm = round_small_nm(pmax);
        const int R = (c.V + kRoundCluster - 1) / kRoundCluster;
        if (base_ok && pm > 0 && c.W * c.k <= 256 && R <= 8 * 256 && static_cast<size_t>(R) * c.d * 4 <= 512 * 1024 &&
            pm * c.d <= 16384 && static_cast<size_t>(pm) * R * 8 <= 64 * 1024) {
            // E streams through two stages: the larger the copies, the faster
            // (one SM's bulk copies complete one after another, at a fixed
            // latency each: about 340 ns, measured on GB300)
            // (each block also keeps its rows of the head weights, 12 F d
            // bytes, where they fit beside stages of at least 32 KB)
            // (larger stages first: they matter more than resident weights)
            if (round_cluster_set_attributes() != cudaSuccess) return DART_ERR_CUDA;
            const size_t cavail = static_cast<size_t>(h->smem_optin) - round_cluster_static_smem(pm);
            int stage = 0;
            bool wres = false;
            size_t smem = 0;
            for (const int stb : {64 * 1024, 48 * 1024, 32 * 1024}) {
                for (const bool wr : {true, false}) {
                    const int st = stb / (c.d * 4) * (c.d * 4);
                    const size_t sm = round_cluster_smem(pm, c.d, R, c.W, c.k, st, wr);
                    if (st > 0 && sm <= cavail) {
                        stage = st;
                        wres = wr;
                        smem = sm;
                        break;
                    }
                }
                if (stage) break;
            }
            if (stage) {
                if (round_cluster_fits(pm, smem)) {
                    h->fused = true;
                    h->fused_cluster = true;
                    h->fused_nm = pm;
                    h->fused_G = kRoundCluster;
                    h->fused_R = R;
                    h->fused_smem = smem;
                    h->fused_ecache = false;
                    h->fused_mstage = false;
                    h->fused_stage = stage;
                    h->fused_wres = wres;
                    return DART_OK;
                }
            }
        }
    }
    const int G = std::min(h->num_sms, 160);
    const int R = (c.V + G - 1) / G;
    const int nm = round_small_nm(nmax);
    bool ok = base_ok && nm > 0 && c.nseq * c.W <= 32 && c.V <= 65536 && c.nseq <= G;
    // each block keeps its E slice for the whole round when it is small
    // (it is read at every depth), and the merge stages a node's lists
    bool ecache = static_cast<size_t>(R) * (c.d + 4) * 4 <= 64 * 1024;
    const bool mstage = static_cast<size_t>(8) * G * c.k * 8 <= 80 * 1024;
    size_t smem = 0;
    if (ok) {
        smem = round_small_smem(nm, c.d, R, c.W, c.k, G, ecache, mstage);
        if (smem > avail && ecache) {
            ecache = false;
            smem = round_small_smem(nm, c.d, R, c.W, c.k, G, ecache, mstage);
        }
        ok = smem <= avail;
    }
    if (ok) {
        if (round_small_set_smem_limits() != cudaSuccess) return DART_ERR_CUDA;
        ok = round_small_blocks_per_sm(nm, smem) >= 1;
    }
    if (!ok) return c.fused_round == DART_ON ? DART_ERR_UNSUPPORTED : DART_OK;
    h->fused = true;
    h->fused_cluster = false;
    h->fused_nm = nm;
    h->fused_G = G;
    h->fused_R = R;
    h->fused_smem = smem;
    h->fused_ecache = ecache;
    h->fused_mstage = mstage;
    return DART_OK;
}

int build_plans(dart_handle* h, const dart_config& c, std::vector<int>& caps, std::vector<DepthPlan>& plans) {
    const bool tc = h->wdtype == DART_BF16;
    caps.assign(c.L + 1, 1);
    for (int i = 1; i <= c.L; i++) caps[i] = std::min(c.W, caps[i - 1] * c.k);
    plans.resize(c.L + 1);
    const int tiles = (c.V + kTileM - 1) / kTileM;
    for (int dep = 1; dep <= c.L; dep++) {
        DepthPlan& p = plans[dep];
        p.P = caps[dep - 1];
        p.N = c.nseq * p.P;
        if (tc) {
            LmheadPlan lp;
            if (!plan_lmhead_tc(p.N, c.V, c.d, c.k, h->num_sms, h->smem_optin, c.lmhead_ctas_per_sm, h->tiled, &lp))
                return DART_ERR_UNSUPPORTED;
            p.NG = lp.NG;
            p.G = lp.G;
            p.nV = lp.nV;
            p.stages = lp.stages;
            p.smem = lp.smem;
            // One group of <= 16 nodes: every CTA streams its own slice of
            // E and the launch is HBM-bound.  Besides the stages it loads
            // before waiting on the previous kernel (which is latency-bound
            // and leaves HBM idle), each CTA then prefetches its next E
            // tiles into L2, about kL2PrefetchBytes over all CTAs.  Measured
            // on GB300 (A/B per round): -0.55 % at d = 4096, -1.0 % at
            // d = 2560, -0.8 % with 16 nodes at d = 2560; with 32 or 64
            // nodes (+2.5 %, +1.0 %) or several groups (+1 %) it is off.
            p.l2pf = (p.G == 1 && p.NG <= 16)
                         ? static_cast<int>(kL2PrefetchBytes / (static_cast<long long>(kTileM) * kBlockK * 2) / p.nV)
                         : 0;
            // The previous depth's selection and head update leave HBM idle
            // for tens of microseconds: a side-stream kernel requests this
            // launch's first E tiles then, as much as L2 holds beside the
            // head weights (6 d^2 bytes, re-read every depth).  Measured on
            // GB300 (tiles per CTA swept, rounds A/B): d = 4096 best near 12
            // of 37 tiles per CTA (-0.55 %), d = 2560 near 20 of 36 (-3.3 %);
            // beyond that it evicts the head weights and costs more than it
            // gains; with several node groups or 32+ nodes it gains nothing.
            const long long free_l2 = h->l2_bytes - 6ll * c.d * c.d;
            const long long per_unit = static_cast<long long>(kTileM) * kBlockK * 2 * p.nV;
            p.epf = (p.l2pf > 0 && free_l2 > 0)
                        ? static_cast<int>(std::min<long long>(free_l2 / per_unit, p.stages + p.l2pf))
                        : 0;
            // The LM-head offers a logit to a node's top-k merges only if it
            // beats the node's filter bound; at k >= 32 the merges of the
            // first tiles (where the bound is still low) limit the kernel,
            // and a small kernel that bounds each node's k-th best score
            // from the rows of largest drafter logit lets the filter start
            // high (csrc/dart_bound.cu).
            // Measured on GB300 (µs per round, same box, AUTO's choice in
            // brackets): 64 nodes, k = 64: 3421 -> 2706 [on]; 64 nodes
            // (4 x 16), k = 16: 2743 -> 2664 [on]; 256 nodes (8 x 32),
            // k = 32: 9594 -> 8670 [on; 128 seed rows: 8964]; 256 nodes,
            // k = 8: 8495 -> 8286 [on]; 32 nodes, k = 32: 2520 -> 2518
            // [off]; 16 nodes, k = 16: 3415 -> 3475 [off].  64- and
            // 128-node groups keep 32 candidate slots per node, which needs
            // the bound (without it: +6 % at 64 nodes, k = 64).
            const int bR = std::max(64, (2 * c.k + 63) / 64 * 64);
            const int bstat = seed_score_static_smem();
            const bool want = c.topk_bound == DART_ON || (c.topk_bound == DART_AUTO && p.N > 32);
            p.bound = (want && c.cand_k == 0 && bR <= kBoundR && c.V >= bR && bstat >= 0 &&
                       seed_score_smem(c.d) + bstat <= static_cast<size_t>(h->smem_optin))
                          ? bR
                          : 0;
        } else {
            p.NG = pick_ng_f32(p.N);
            p.G = (p.N + p.NG - 1) / p.NG;
            p.nV = std::max(1, std::min(h->num_sms / p.G, tiles));
            // fewer vocabulary tiles than SMs: clusters of DS blocks split d
            // (toy shape, V = 4096: 32 tiles x 4 slices of d = 256)
            p.f32_ds = 1;
            while (p.f32_ds < 8 && 2 * p.f32_ds <= c.d / kBlockK && p.nV * p.G * 2 * p.f32_ds <= h->num_sms)
                p.f32_ds *= 2;
            p.stages = 0;
            p.l2pf = 0;
            p.epf = 0;
            p.bound = 0;
            p.smem = lmhead_f32_smem(p.NG, c.k);
            if (p.smem > h->smem_optin) return DART_ERR_UNSUPPORTED;
        }
        p.nlist = c.cand_k > 0 ? c.cand_k : p.nV;  // one single-key list per candidate of C_d
        p.klist = c.cand_k > 0 ? 1 : c.k;
        p.cand_ds = 0;
        if (c.cand_k > 0) {
            p.cand_ds = cand_score_slices(p.P, c.d, c.nseq, c.cand_k, h->smem_optin);
            if (p.cand_ds == 0) return DART_ERR_UNSUPPORTED;
        }
        p.Pn = caps[dep];
        p.Nc = c.nseq * p.Pn;
        p.split = p.side = 0;
        if (dep < c.L) {
            // Split first head layer (bf16 weights):
            //   W_i . [h_p ; E[t_c]] = W_i[:, 0:d] . h_p + Q[t_c],
            // Q = the per-token table computed once per handle.  The GEMM then
            // runs over the parents' states, which are already held as hi/lo
            // rows (no gather of the inputs), with half of W_i, beside the
            // selection of the children, and Q[t_c] is added in the SiLU
            // kernel.  head_split = DART_OFF turns it off; head_split_stream =
            // DART_OFF runs its GEMM after merge + select on the same stream.
            p.split = (tc && c.head_split != DART_OFF) ? 1 : 0;
            p.side = (p.split && c.head_split_stream != DART_OFF) ? 1 : 0;
            p.g1 = p.split ? gemm_plan(h, c.d, p.N, c.d / kBlockK, tc) : gemm_plan(h, 2 * c.d, p.Nc, c.d / kBlockK, tc);
            p.g2 = gemm_plan(h, c.d, p.Nc, c.d / kBlockK, tc);
            if (tc) {
                // two CTAs per SM when both fit with >= 4 stages: twice the
                // independent weight streams, k split twice as finely
                // (the split layer's GEMM runs over the parents, fewer nodes
                // than the W_o GEMM's children: size both for the larger group)
                const int ngmax = std::max(p.g1.NG, p.g2.NG);
                const int sb = tc_stage_bytes(ngmax);
                const int st2 = std::min(tc_stages(h->smem_optin / 2 - 2048, sb, gemm_tc_fixed_smem(16)), 8);
                const int smem2 = gemm_tc_fixed_smem(st2) + st2 * sb;
                int cps = 1;
                if (st2 >= 4 && gemm_tc_ctas_per_sm(ngmax, smem2) >= 2) {
                    cps = 2;
                    p.g1.stages = st2;
                } else {
                    p.g1.stages = std::min(tc_stages(h->smem_optin, sb, gemm_tc_fixed_smem(16)), 8);
                }
                p.g2.stages = p.g1.stages;
                if (p.g1.stages < 2) return DART_ERR_UNSUPPORTED;
                p.g1_smem = gemm_tc_fixed_smem(p.g1.stages) + p.g1.stages * sb;
                p.g2_smem = p.g1_smem;
                // One node group of <= 16 nodes: k split over every resident
                // CTA, partial tiles summed by the SiLU / residual-norm kernels
                // (the small kernel between the GEMMs is where the W_o GEMM's
                // CTAs become resident and fetch their first weight tiles).
                // Larger node sets: the k splits of a tile are one cluster
                // (the largest <= 8 whose clusters all fit on the GPU at
                // once) and are summed on chip, with SiLU applied there (the
                // split layer's GEMM writes the plain sum; SiLU follows the
                // addition of Q[t_c]).
                const bool cluster = p.Nc > 16;
                const bool cluster1 = p.split ? p.N > 16 : cluster;
                for (GemmArgs* g : {&p.g1, &p.g2}) {
                    const int tiles_mg = g->MT * g->G;
                    const int cap = cps * h->num_sms;
                    const bool cl = g == &p.g1 ? cluster1 : cluster;
                    if (cl) {
                        int sc = std::max(1, std::min({kMaxClusterK, g->KB, cap / tiles_mg}));
                        for (; sc > 1; sc--)
                            if (gemm_tc_max_clusters(g->NG, p.g1_smem, sc) >= tiles_mg) break;
                        g->S = sc;
                    } else {
                        g->S = std::max(1, std::min(g->KB, cap / tiles_mg));
                    }
                }
                p.g1.mode = cluster1 ? (p.split ? kGemmSum : kGemmSiluSplit) : kGemmPartials;
                p.g2.mode = cluster ? kGemmSum : kGemmPartials;
                p.g1.a_tiled_kb = h->wtiled ? h->Kwi / kBlockK : 0;
                p.g2.a_tiled_kb = h->wtiled ? c.d / kBlockK : 0;
                // Candidate-restricted scoring streams nothing through L2
                // between the depths: with <= 16 children (weight-bound
                // GEMMs) the largest of {W_i and W_o, W_i (4 d^2 bytes, 2 d^2
                // for the split layer), W_o (2 d^2)} within kL2KeepBytes is
                // loaded evict-last and read from HBM once per round instead
                // of once per depth.
                // Measured on GB300 (A/B, K = 64): d = 2560, both (39 MB):
                // -4.9 % per round; d = 4096: W_i (67 MB) -6.0 %, W_o
                // (34 MB) -2.0 %, both (101 MB) +2.1 %; W_o with 256 children
                // (cluster GEMMs) +0.8 %.
                const long long wo_bytes = 2ll * c.d * c.d, wi_bytes = (p.split ? 2ll : 4ll) * c.d * c.d;
                p.g1.keep_a = p.g2.keep_a = 0;
                if (c.cand_k > 0 && !cluster) {
                    if (wi_bytes + wo_bytes <= kL2KeepBytes)
                        p.g1.keep_a = p.g2.keep_a = 1;
                    else if (wi_bytes <= kL2KeepBytes)
                        p.g1.keep_a = 1;
                    else if (wo_bytes <= kL2KeepBytes)
                        p.g2.keep_a = 1;
                }
            }
        }
    }
    return DART_OK;
}

size_t max_part_floats(const dart_handle* h) {
    size_t m = 1;
    for (const std::vector<DepthPlan>* ps : {&h->plans, &h->cplans})
        for (int dep = 1; dep + 1 < static_cast<int>(ps->size()); dep++) {
            const DepthPlan& p = (*ps)[dep];
            m = std::max(m, static_cast<size_t>(p.g1.S) * std::max(p.N, p.Nc) * h->cfg.d);
            m = std::max(m, static_cast<size_t>(p.g2.S) * p.Nc * h->cfg.d);
        }
    return m;
}

int alloc_workspace(dart_handle* h) {
    const dart_config& c = h->cfg;
    const size_t d = c.d;
    int rc = DART_OK;
    size_t max_nvn = 1, max_keys = 1;  // key lists x nodes; keys incl. one padding key per node
    for (const std::vector<DepthPlan>* ps : {&h->plans, &h->cplans})
        for (int dep = 1; dep < static_cast<int>(ps->size()); dep++) {
            const DepthPlan& p = (*ps)[dep];
            max_nvn = std::max(max_nvn, static_cast<size_t>(p.nlist) * p.N);
            max_keys = std::max(max_keys, (static_cast<size_t>(p.nlist) * p.klist + 1) * p.N);
        }
    const size_t super = static_cast<size_t>(c.nseq) * c.L * c.W;
#define DART_ALLOC(ptr, n) \
    if (rc == DART_OK) rc = dalloc(h, &(ptr), (n));
    DART_ALLOC(h->hbuf[0], kNPadMax * d)
    DART_ALLOC(h->hbuf[1], kNPadMax * d)
    if (h->wdtype == DART_BF16) {
        DART_ALLOC(h->HL, 2 * kNPadMax * d)
        DART_ALLOC(h->XL, 2 * kNPadMax * 2 * d)
        DART_ALLOC(h->AL, 2 * kNPadMax * d)
    } else {
        DART_ALLOC(h->X32, kNPadMax * 2 * d)
        DART_ALLOC(h->A32, kNPadMax * d)
    }
    DART_ALLOC(h->part, max_part_floats(h))
    DART_ALLOC(h->part_ms, max_nvn)
    DART_ALLOC(h->part_key, max_keys)  // part_stride(nlist, klist) keys per node
    DART_ALLOC(h->node_logq, static_cast<size_t>(kNPadMax) * c.k)
    DART_ALLOC(h->node_tok, static_cast<size_t>(kNPadMax) * c.k)
    DART_ALLOC(h->node_lse, kNPadMax)
    DART_ALLOC(h->tree_tok, super)
    DART_ALLOC(h->tree_parent, super)
    DART_ALLOC(h->tree_score, super)
    DART_ALLOC(h->tree_count, static_cast<size_t>(c.nseq) * c.L)
    DART_ALLOC(h->child_prow, kNPadMax)
    DART_ALLOC(h->child_tok, kNPadMax)
    DART_ALLOC(h->seq_ticket, c.nseq)
    DART_ALLOC(h->status, 1)
    DART_ALLOC(h->gthr, static_cast<size_t>(c.L) * kNPadMax)
    if (h->wdtype == DART_BF16) DART_ALLOC(h->bound_y, static_cast<size_t>(kNPadMax) * kBoundR)
    bool any_split = false;
    for (int dep = 1; dep < c.L; dep++) any_split = any_split || h->plans[dep].split;
    if (any_split) DART_ALLOC(h->Qtab, static_cast<size_t>(c.V) * d)
    if (h->tiled) DART_ALLOC(h->Et, static_cast<size_t>((c.V + kTileM - 1) / kTileM) * kTileM * d)
    if (h->wtiled) {
        DART_ALLOC(h->Wit, static_cast<size_t>((c.d + kTileM - 1) / kTileM) * kTileM * h->Kwi)
        DART_ALLOC(h->Wot, static_cast<size_t>((c.d + kTileM - 1) / kTileM) * kTileM * d)
    }
    if (h->fused) {
        const size_t nc = static_cast<size_t>(c.nseq) * c.W, G = h->fused_G;
        DART_ALLOC(h->f_rbuf, nc * d)
        DART_ALLOC(h->f_abuf, nc * d)
        DART_ALLOC(h->f_ssqp, nc * G)
        DART_ALLOC(h->f_pms, nc * G)
        DART_ALLOC(h->f_pkey, nc * G * c.k)
        DART_ALLOC(h->f_bar, kRoundBarWords)
        DART_ALLOC(h->f_abort, 1)
    }
    const size_t ns = c.nseq, Bp = h->Bp, S1 = static_cast<size_t>(c.B) + 1;
    if (c.variants & DART_VARIANT_CHAIN_DDTREE) {
        DART_ALLOC(h->zrows, ns * c.L * c.V)
        DART_ALLOC(h->chain_lse, ns * c.L)
        DART_ALLOC(h->ddt_tok, ns * c.L * Bp)
        DART_ALLOC(h->ddt_z, ns * c.L * Bp)
        DART_ALLOC(h->ddt_part, ns * c.L * h->ddt_S * Bp)
        DART_ALLOC(h->ddt_ticket, ns * c.L)
    }
    if (c.variants & DART_VARIANT_SEQ_HEAP) {
        DART_ALLOC(h->sh_tab, ns * S1 * d)
        DART_ALLOC(h->sh_ltok, ns * S1 * Bp)
        DART_ALLOC(h->sh_lz, ns * S1 * Bp)
        DART_ALLOC(h->sh_llse, ns * S1)
        DART_ALLOC(h->sh_next, ns * S1)
        DART_ALLOC(h->sh_offer, ns * S1)
        DART_ALLOC(h->sh_npop, ns)
        DART_ALLOC(h->sh_dlog_row, ns)
        DART_ALLOC(h->sh_zrow, ns * c.V)
        DART_ALLOC(h->sh_part, ns * h->sh_S * Bp)
        DART_ALLOC(h->sh_ticket, ns)
    }
    if (c.cand_k > 0) {
        size_t scr = 1;
        for (int dep = 1; dep <= c.L; dep++)
            scr = std::max(scr, static_cast<size_t>(h->plans[dep].cand_ds) * h->plans[dep].N * c.cand_k);
        DART_ALLOC(h->cand_tok, static_cast<size_t>(c.nseq) * c.L * c.cand_k)
        DART_ALLOC(h->cand_scratch, scr)
        DART_ALLOC(h->cand_ticket, static_cast<size_t>(c.nseq) * ((c.cand_k + 7) / 8))
        DART_ALLOC(h->cand_part, static_cast<size_t>(c.nseq) * c.L *
                                     cand_topk_slices(c.V, c.cand_k, c.nseq * c.L, h->num_sms) * c.cand_k)
        DART_ALLOC(h->cand_rticket, static_cast<size_t>(c.nseq) * c.L)
    }
#undef DART_ALLOC
    if (rc != DART_OK) return rc;
    // zeroed once: stale rows of the operand buffers are always finite
    for (void* p : {static_cast<void*>(h->hbuf[0]), static_cast<void*>(h->hbuf[1])})
        if (cudaMemset(p, 0, kNPadMax * d * sizeof(float)) != cudaSuccess) return DART_ERR_CUDA;
    if (h->wdtype == DART_BF16) {
        if (cudaMemset(h->HL, 0, 2 * kNPadMax * d * 2) != cudaSuccess) return DART_ERR_CUDA;
        if (cudaMemset(h->XL, 0, 2 * kNPadMax * 2 * d * 2) != cudaSuccess) return DART_ERR_CUDA;
        if (cudaMemset(h->AL, 0, 2 * kNPadMax * d * 2) != cudaSuccess) return DART_ERR_CUDA;
    } else {
        if (cudaMemset(h->X32, 0, kNPadMax * 2 * d * 4) != cudaSuccess) return DART_ERR_CUDA;
        if (cudaMemset(h->A32, 0, kNPadMax * d * 4) != cudaSuccess) return DART_ERR_CUDA;
    }
    if (cudaMemset(h->seq_ticket, 0, c.nseq * sizeof(int)) != cudaSuccess) return DART_ERR_CUDA;
    if (cudaMemset(h->status, 0, sizeof(int)) != cudaSuccess) return DART_ERR_CUDA;
    if (cudaMemset(h->tree_count, 0, c.nseq * c.L * sizeof(int)) != cudaSuccess) return DART_ERR_CUDA;
    if (h->ddt_ticket && cudaMemset(h->ddt_ticket, 0, ns * c.L * sizeof(int)) != cudaSuccess) return DART_ERR_CUDA;
    if (h->sh_ticket && cudaMemset(h->sh_ticket, 0, ns * sizeof(int)) != cudaSuccess) return DART_ERR_CUDA;
    if (h->fused && (cudaMemset(h->f_bar, 0, kRoundBarWords * sizeof(unsigned)) != cudaSuccess ||
                     cudaMemset(h->f_abort, 0, sizeof(int)) != cudaSuccess ||
                     round_small_set_smem_limits() != cudaSuccess ||
                     (h->fused_cluster && round_cluster_set_attributes() != cudaSuccess)))
        return DART_ERR_CUDA;
    // one-time kernel attributes
    int max_sel = 0;
    for (int dep = 1; dep <= c.L; dep++)
        max_sel = std::max(max_sel, merge_select_smem(h->plans[dep].nlist, h->plans[dep].klist, c.k, c.W));
    if (max_sel > h->smem_optin) return DART_ERR_UNSUPPORTED;
    if (select_set_smem_limits() != cudaSuccess) return DART_ERR_CUDA;
    if (c.cand_k > 0) {
        for (int dep = 1; dep <= c.L; dep++)
            if (cand_score_smem(h->plans[dep].P, c.d, h->plans[dep].cand_ds) > h->smem_optin - 1024)
                return DART_ERR_UNSUPPORTED;
        if (cudaMemset(h->cand_ticket, 0, c.nseq * ((c.cand_k + 7) / 8) * sizeof(int)) != cudaSuccess ||
            cudaMemset(h->cand_rticket, 0, static_cast<size_t>(c.nseq) * c.L * sizeof(int)) != cudaSuccess)
            return DART_ERR_CUDA;
    }
    if ((c.cand_k > 0 || c.variants) && cand_set_smem_limits() != cudaSuccess) return DART_ERR_CUDA;
    if ((c.variants & DART_VARIANT_CHAIN_DDTREE) && heap_set_smem_limits() != cudaSuccess) return DART_ERR_CUDA;
    if (h->wdtype == DART_BF16) {
        if (tc_set_smem_limits(h->smem_optin) != cudaSuccess) return DART_ERR_CUDA;
        if (seed_score_set_smem_limit(h->smem_optin) != cudaSuccess) return DART_ERR_CUDA;
    } else {
        if (f32_set_smem_limits(h->smem_optin) != cudaSuccess) return DART_ERR_CUDA;
    }
    return DART_OK;
}

int make_tensor_maps(dart_handle* h) {
    const dart_config& c = h->cfg;
    const uint64_t d = c.d;
    // the LM-head's E: [V][d] row-major, or the tiled copy viewed as rows of 64
    // elements (tile (rt, kb) = rows (rt * d/64 + kb) * 128 .. + 127)
    auto tiled_rows = [](uint64_t rows, uint64_t cols) {
        return (rows + kTileM - 1) / kTileM * kTileM * (cols / kBlockK);
    };
    bool ok = (h->tiled ? encode_bf16_2d(&h->tmE, h->Et, kBlockK, tiled_rows(c.V, d), kTileM)
                        : encode_bf16_2d(&h->tmE, h->E, d, c.V, kTileM)) &&
              (h->wtiled ? encode_bf16_2d(&h->tmWi, h->Wit, kBlockK, tiled_rows(d, h->Kwi), kTileM) &&
                               encode_bf16_2d(&h->tmWo, h->Wot, kBlockK, tiled_rows(d, d), kTileM)
                         : encode_bf16_2d(&h->tmWi, h->Wi, 2 * d, d, kTileM) &&
                               encode_bf16_2d(&h->tmWo, h->Wo, d, d, kTileM));
    const int ngs[3] = {16, 32, 64};
    for (int i = 0; i < 3 && ok; i++) {
        ok = encode_bf16_2d(&h->tmH[i], h->HL, d, 2 * kNPadMax, ngs[i]) &&
             encode_bf16_2d(&h->tmX[i], h->XL, 2 * d, 2 * kNPadMax, ngs[i]) &&
             encode_bf16_2d(&h->tmA[i], h->AL, d, 2 * kNPadMax, ngs[i]);
    }
    if (ok) ok = encode_bf16_2d(&h->tmH[3], h->HL, d, 2 * kNPadMax, 128);  // LM-head 128-node groups
    if (ok && h->Qtab) {
        ok = encode_bf16_2d(&h->tmWiR, static_cast<const __nv_bfloat16*>(h->Wi) + d, d, d, kTileM, 2 * d) &&
             encode_bf16_2d(&h->tmEB, h->E, d, c.V, 64);
    }
    return ok ? DART_OK : DART_ERR_UNSUPPORTED;
}

// Q[t][j] = sum_k W_i[j][d + k] * E[t][k] for every token t: one launch of
// the head GEMM kernel with the roles of the operands swapped (A = the
// second half of W_i, M = d output features; B = E, V rows as nodes in
// groups of 64, no lo half since E is exact in bf16), k not split, so its
// partial tile is the result, written as [V][d].
int compute_qtab(dart_handle* h, cudaStream_t st) {
    const dart_config& c = h->cfg;
    GemmArgs q;
    std::memset(&q, 0, sizeof q);
    q.M = c.d;
    q.K = c.d;
    q.N = c.V;
    q.NG = 64;
    q.G = (c.V + 63) / 64;
    q.MT = (c.d + kTileM - 1) / kTileM;
    q.S = 1;
    q.KB = c.d / kBlockK;
    q.lo_kb_end = 0;
    q.bhalf = 0;
    const int sb = tc_stage_bytes(64);
    const int st2 = std::min(tc_stages(h->smem_optin / 2 - 2048, sb, gemm_tc_fixed_smem(16)), 8);
    q.stages = st2 >= 3 ? st2 : std::min(tc_stages(h->smem_optin, sb, gemm_tc_fixed_smem(16)), 8);
    if (q.stages < 2) return DART_ERR_UNSUPPORTED;
    q.mode = kGemmPartials;
    q.keep_a = 1;  // the 2 d^2-byte A operand is read by every node group
    q.out = h->Qtab;
    q.status = h->status;
    const int smem = gemm_tc_fixed_smem(q.stages) + q.stages * sb;
    return cuda_err(launch_gemm_tc(&h->tmWiR, &h->tmEB, q, smem, st));
}

void release(dart_handle* h) {
    for (auto& g : h->graphs) cudaGraphExecDestroy(g.exec);
    h->graphs.clear();
    for (cudaEvent_t e : h->ev) cudaEventDestroy(e);
    h->ev.clear();
    if (h->cap_stream) cudaStreamDestroy(h->cap_stream);
    h->cap_stream = nullptr;
    if (h->side) cudaStreamDestroy(h->side);
    h->side = nullptr;
    if (h->ev_fork) cudaEventDestroy(h->ev_fork);
    if (h->ev_join) cudaEventDestroy(h->ev_join);
    h->ev_fork = h->ev_join = nullptr;
    for (void* p : h->allocs) cudaFree(p);
    h->allocs.clear();
}

// ---------------------------------------------------------------- enqueue

enum Kind {
    kLmhead = 0, kSelect, kGather, kGemm1, kSilu, kGemm2, kNorm, kPrep, kEmit, kCandTopk, kCandScore, kGatherSilu,
    kRowTopk, kDdtree, kSeqStep, kSeqEmit, kFusedRound, kL2Prefetch, kBound, kNumKinds
};

// Opens an event pair around the next launch when profiling (no-op otherwise).
int prof_begin(dart_handle* h, int kind, cudaStream_t st) {
    if (!h->profiling || h->ev_used + 2 > kMaxProfilePairs * 2) return -1;
    while (static_cast<int>(h->ev.size()) < h->ev_used + 2) {
        cudaEvent_t e;
        if (cudaEventCreate(&e) != cudaSuccess) return -1;
        h->ev.push_back(e);
        h->ev_kind.push_back(-1);
    }
    const int i = h->ev_used;
    h->ev_kind[i] = kind;
    cudaEventRecord(h->ev[i], st);
    return i;
}
void prof_end(dart_handle* h, int i, cudaStream_t st) {
    if (i < 0) return;
    cudaEventRecord(h->ev[i + 1], st);
    h->ev_used = i + 2;
}

// LM-head launch arguments of plan p (drafter row and cross-CTA bounds are
// set by the caller); h32: the nodes' fp32 states (fp32 weights).
LmheadArgs lmhead_args(const dart_handle* h, const dart_config& c, const DepthPlan& p, const float* dlog,
                       const float* h32) {
    LmheadArgs la;
    std::memset(&la, 0, sizeof la);
    la.V = c.V;
    la.d = c.d;
    la.N = p.N;
    la.NG = p.NG;
    la.G = p.G;
    la.nV = p.nV;
    la.k = c.k;
    la.tiles = (c.V + kTileM - 1) / kTileM;
    la.P = p.P;
    la.invT = c.temperature > 0.0f ? 1.0f / c.temperature : 1.0f;
    la.dlog = dlog;
    la.dlog_seq_stride = static_cast<long long>(c.L) * c.V;
    la.bhalf = kNPadMax;
    la.stages = p.stages;
    la.l2pf = p.l2pf;
    la.part_ms = h->part_ms;
    la.part_key = h->part_key;
    la.status = h->status;
    la.h32 = h32;
    la.E32 = static_cast<const float*>(h->E);
    la.e_tiled = h->Et ? 1 : 0;
    la.DS = p.f32_ds > 0 ? p.f32_ds : 1;
    return la;
}

// Merge + frontier-selection launch arguments of plan p at depth dep.
SelectArgs select_args(const dart_handle* h, const dart_config& c, const DepthPlan& p, int dep) {
    SelectArgs sa;
    std::memset(&sa, 0, sizeof sa);
    sa.N = p.N;
    sa.P = p.P;
    sa.k = c.k;
    sa.nV = p.nlist;
    sa.klist = p.klist;
    sa.W = c.W;
    sa.L = c.L;
    sa.nseq = c.nseq;
    sa.dep = dep;
    sa.Pn = p.Pn;
    sa.beta = c.beta;
    sa.part_ms = h->part_ms;
    sa.part_key = h->part_key;
    sa.node_logq = h->node_logq;
    sa.node_tok = h->node_tok;
    sa.node_lse = h->node_lse;
    sa.tree_tok = h->tree_tok;
    sa.tree_parent = h->tree_parent;
    sa.tree_score = h->tree_score;
    sa.tree_count = h->tree_count;
    sa.child_prow = h->child_prow;
    sa.child_tok = h->child_tok;
    sa.seq_ticket = h->seq_ticket;
    sa.status = h->status;
    return sa;
}

// Optional outputs of one depth (the chain of Domino-chain + DDTree): every
// node's scaled logits z[n][v] -> zout[n * zout_stride + v], and its
// log-sum-exp -> lse_hist[n * lse_hist_stride].
struct DepthOutputs {
    float* zout;
    long long zout_stride;
    float* lse_hist;
    long long lse_hist_stride;
};

int enqueue_head_update(dart_handle* h, const dart_config& c, const DepthPlan& p, const float* hcur, float* hnext,
                        bool g1_launched, cudaStream_t st);

// Algorithm 1, one iteration, for configuration c with plans `plans` (the
// handle's, or the one-node-per-sequence chain's).
int enqueue_depth(dart_handle* h, const dart_config& c, const std::vector<DepthPlan>& plans, int dep,
                  const float* dlog, const float* anchor, cudaStream_t st, const DepthOutputs* outs = nullptr) {
    const DepthPlan& p = plans[dep];
    const bool tc = h->wdtype == DART_BF16;
    cudaError_t e = cudaSuccess;
    if (dep == 1) {
        const int pi = prof_begin(h, kPrep, st);
        e = launch_prep_anchor(anchor, c.nseq, c.d, h->hbuf[0], tc ? h->HL : nullptr, kNPadMax, h->gthr,
                               c.L * kNPadMax, st);
        prof_end(h, pi, st);
        if (e != cudaSuccess) return DART_ERR_CUDA;
        h->cur = 0;
        if (c.cand_k > 0) {
            // C_d = TopK(L_d^base, K) of every position of every sequence
            const int pc = prof_begin(h, kCandTopk, st);
            const int rows = c.nseq * c.L;
            e = launch_cand_topk(dlog, rows, c.V, c.cand_k, cand_topk_slices(c.V, c.cand_k, rows, h->num_sms),
                                 h->cand_tok, h->cand_part, h->cand_rticket, st);
            prof_end(h, pc, st);
            if (e != cudaSuccess) return DART_ERR_CUDA;
        }
    }
    // 1) LM-head scoring of every prefix in S_{dep-1} (fused log-sum-exp / top-k)
    LmheadArgs la = lmhead_args(h, c, p, dlog, h->hbuf[h->cur]);
    la.dlog_row_off = static_cast<long long>(dep - 1) * c.V;
    la.gthr = h->gthr + static_cast<size_t>(dep - 1) * kNPadMax;
    if (outs) {
        la.zout = outs->zout;
        la.zout_stride = outs->zout_stride;
    }
    int pi;
    if (c.cand_k > 0) {
        // candidate-restricted scoring: every node against its sequence's C_d
        CandArgs ca;
        std::memset(&ca, 0, sizeof ca);
        ca.K = c.cand_k;
        ca.P = p.P;
        ca.d = c.d;
        ca.L = c.L;
        ca.dep = dep;
        ca.nseq = c.nseq;
        ca.wbf16 = tc ? 1 : 0;
        ca.V = c.V;
        ca.invT = la.invT;
        ca.cand_tok = h->cand_tok;
        ca.dlog = dlog;
        ca.dlog_seq_stride = la.dlog_seq_stride;
        ca.dlog_row_off = la.dlog_row_off;
        ca.h = h->hbuf[h->cur];
        ca.E = h->E;
        ca.part_ms = h->part_ms;
        ca.part_key = h->part_key;
        ca.DS = p.cand_ds;
        ca.scratch = h->cand_scratch;
        ca.ticket = h->cand_ticket;
        pi = prof_begin(h, kCandScore, st);
        e = launch_cand_score(ca, st);
    } else {
        if (p.bound) {
            BoundArgs ba;
            std::memset(&ba, 0, sizeof ba);
            ba.P = p.P;
            ba.d = c.d;
            ba.V = c.V;
            ba.k = c.k;
            ba.R = p.bound;
            ba.invT = la.invT;
            ba.h = h->hbuf[h->cur];
            ba.E = static_cast<const __nv_bfloat16*>(h->E);
            ba.dlog = dlog;
            ba.dlog_seq_stride = la.dlog_seq_stride;
            ba.dlog_row_off = la.dlog_row_off;
            ba.ybuf = h->bound_y;
            ba.status = h->status;
            const int pb = prof_begin(h, kBound, st);
            e = launch_seed_score(ba, c.nseq, st);
            prof_end(h, pb, st);
            if (e != cudaSuccess) return DART_ERR_CUDA;
            la.seed_y = h->bound_y;
            la.seed_R = p.bound;
        }
        pi = prof_begin(h, kLmhead, st);
        e = tc ? launch_lmhead_tc(&h->tmE, &h->tmH[ng_index(p.NG)], la, p.smem, st) : launch_lmhead_f32(la, st);
    }
    prof_end(h, pi, st);
    if (e != cudaSuccess) return DART_ERR_CUDA;
    if (p.side) {
        // Split first head layer: U = W_i[:, 0:d] . h over the parents needs
        // only their states (the hi/lo rows the LM-head just read), so it runs
        // on the side stream while merge + select finds the children; it
        // writes `part`, whose last reader (residual_norm of the previous
        // depth) finished before the LM-head did.  Joined before gather_silu.
        GemmArgs g1 = p.g1;
        g1.out = h->part;
        g1.outL = h->AL;
        g1.status = h->status;
        if (cudaEventRecord(h->ev_fork, st) != cudaSuccess || cudaStreamWaitEvent(h->side, h->ev_fork, 0) != cudaSuccess)
            return DART_ERR_CUDA;
        // HBM idles while the children are selected: the next LM-head's
        // first E tiles (its L2-prefetch window) are requested now, beside it
        if (c.cand_k == 0 && dep < c.L && plans[dep + 1].epf > 0) {
            const DepthPlan& q = plans[dep + 1];
            pi = prof_begin(h, kL2Prefetch, h->side);
            e = launch_lmhead_l2_prefetch(&h->tmE, (c.V + kTileM - 1) / kTileM, q.nV, c.d, q.epf, h->Et ? 1 : 0,
                                          h->side);
            prof_end(h, pi, h->side);
            if (e != cudaSuccess) return DART_ERR_CUDA;
        }
        pi = prof_begin(h, kGemm1, h->side);
        e = launch_gemm_tc(&h->tmWi, &h->tmH[ng_index(g1.NG)], g1, p.g1_smem, h->side);
        prof_end(h, pi, h->side);
        if (e != cudaSuccess || cudaEventRecord(h->ev_join, h->side) != cudaSuccess) return DART_ERR_CUDA;
    }
    // 2) merge partials, log q~, Eq. 5 scores, global top-W -> S_dep
    SelectArgs sa = select_args(h, c, p, dep);
    sa.gthr = c.cand_k > 0 ? nullptr : la.gthr;
    if (outs) {
        sa.lse_hist = outs->lse_hist;
        sa.lse_hist_stride = outs->lse_hist_stride;
    }
    pi = prof_begin(h, kSelect, st);
    e = launch_merge_select(sa, st);
    prof_end(h, pi, st);
    if (e != cudaSuccess) return DART_ERR_CUDA;
    h->last_rows = p.N;
    if (dep == c.L) return DART_OK;
    // 3) correction-head update of the retained children (Algorithm 1, state update)
    const int rc = enqueue_head_update(h, c, p, h->hbuf[h->cur], h->hbuf[1 - h->cur], p.side != 0, st);
    if (rc != DART_OK) return rc;
    h->cur = 1 - h->cur;
    h->last_rows = p.Nc;
    return DART_OK;
}

// Correction-head update of the children listed in child_prow / child_tok
// (Algorithm 1, "update their states"): hnext[c] = RMSNorm(hcur[prow[c]] +
// W_o SiLU(W_i [hcur[prow[c]] ; E[tok[c]]])), with the hi/lo bf16 split of
// the result in HL.  With the split first layer the W_i[:, 0:d] GEMM reads
// the parents' hi/lo rows in HL; g1_launched: it already runs on the side
// stream (joined here).
int enqueue_head_update(dart_handle* h, const dart_config& c, const DepthPlan& p, const float* hcur, float* hnext,
                        bool g1_launched, cudaStream_t st) {
    const bool tc = h->wdtype == DART_BF16;
    cudaError_t e = cudaSuccess;
    int pi;
    if (!tc && head_small_f32_slices(c.d) > 0) {
        // small fp32 heads: the whole update in one launch (one cluster per child)
        pi = prof_begin(h, kNorm, st);
        e = launch_head_small_f32(p.Nc, c.d, h->child_prow, h->child_tok, hcur, static_cast<const float*>(h->E),
                                  static_cast<const float*>(h->Wi), static_cast<const float*>(h->Wo), c.rms_eps, hnext,
                                  st);
        prof_end(h, pi, st);
        return e == cudaSuccess ? DART_OK : DART_ERR_CUDA;
    }
    if (!p.split) {
        pi = prof_begin(h, kGather, st);
        e = launch_gather_x(p.Nc, c.d, h->child_prow, h->child_tok, hcur, h->E, tc ? 1 : 0, h->XL, kNPadMax, h->X32,
                            st);
        prof_end(h, pi, st);
        if (e != cudaSuccess) return DART_ERR_CUDA;
    }
    GemmArgs g1 = p.g1, g2 = p.g2;
    g1.out = h->part;
    g1.outL = h->AL;
    g2.out = h->part;
    g1.status = g2.status = h->status;
    if (!g1_launched) {  // (on the side stream it was launched after the LM-head)
        pi = prof_begin(h, kGemm1, st);
        if (p.split) {
            e = launch_gemm_tc(&h->tmWi, &h->tmH[ng_index(g1.NG)], g1, p.g1_smem, st);
        } else if (tc) {
            e = launch_gemm_tc(&h->tmWi, &h->tmX[ng_index(g1.NG)], g1, p.g1_smem, st);
        } else {
            g1.A32 = static_cast<const float*>(h->Wi);
            g1.B32 = h->X32;
            e = launch_gemm_f32(g1, st);
        }
        prof_end(h, pi, st);
        if (e != cudaSuccess) return DART_ERR_CUDA;
    }
    const bool fused = tc && g1.mode != kGemmPartials;  // SiLU applied in the GEMM's cluster reduction
    if (p.split) {
        if (g1_launched && cudaStreamWaitEvent(st, h->ev_join, 0) != cudaSuccess) return DART_ERR_CUDA;
        pi = prof_begin(h, kGatherSilu, st);
        // (a cluster GEMM wrote the summed U: one "split")
        e = launch_gather_silu(p.Nc, c.d, g1.mode == kGemmPartials ? g1.S : 1, g1.N, h->part, h->child_prow,
                               h->child_tok, c.V, h->Qtab, h->AL, kNPadMax, h->status, st);
        prof_end(h, pi, st);
        if (e != cudaSuccess) return DART_ERR_CUDA;
    } else if (!fused) {
        pi = prof_begin(h, kSilu, st);
        e = launch_silu_split(p.Nc, c.d, g1.S, h->part, tc ? h->AL : nullptr, kNPadMax, h->A32, st);
        prof_end(h, pi, st);
        if (e != cudaSuccess) return DART_ERR_CUDA;
    }
    pi = prof_begin(h, kGemm2, st);
    if (tc) {
        e = launch_gemm_tc(&h->tmWo, &h->tmA[ng_index(g2.NG)], g2, p.g2_smem, st);
    } else {
        g2.A32 = static_cast<const float*>(h->Wo);
        g2.B32 = h->A32;
        e = launch_gemm_f32(g2, st);
    }
    prof_end(h, pi, st);
    if (e != cudaSuccess) return DART_ERR_CUDA;
    pi = prof_begin(h, kNorm, st);
    const int s2 = tc && g2.mode != kGemmPartials ? 1 : g2.S;  // the W_o cluster GEMM wrote the sum
    e = launch_residual_norm(p.Nc, c.d, s2, h->part, h->child_prow, hcur, c.rms_eps, hnext, tc ? h->HL : nullptr,
                             kNPadMax, st);
    prof_end(h, pi, st);
    return e == cudaSuccess ? DART_OK : DART_ERR_CUDA;
}

int check_out(const dart_tree_out* o) {
    if (!o || !o->tokens || !o->parents || !o->depths || !o->pos_ids || !o->scores || !o->n_nodes || !o->mask)
        return DART_ERR_INVALID;
    if (!aligned4(o->tokens) || !aligned4(o->parents) || !aligned4(o->depths) || !aligned4(o->pos_ids) ||
        !aligned4(o->scores) || !aligned4(o->n_nodes) || (reinterpret_cast<uintptr_t>(o->mask) & 7u))
        return DART_ERR_INVALID;
    return DART_OK;
}

EmitArgs emit_args(const dart_handle* h, const dart_tree_out* o) {
    const dart_config& c = h->cfg;
    EmitArgs a;
    a.L = c.L;
    a.W = c.W;
    a.B = c.B;
    a.nseq = c.nseq;
    a.pos_offset = c.pos_offset;
    a.tree_tok = h->tree_tok;
    a.tree_parent = h->tree_parent;
    a.tree_score = h->tree_score;
    a.tree_count = h->tree_count;
    a.tokens = o->tokens;
    a.parents = o->parents;
    a.depths = o->depths;
    a.pos_ids = o->pos_ids;
    a.n_nodes = o->n_nodes;
    a.scores = o->scores;
    a.mask = o->mask;
    a.status = h->status;
    return a;
}

int enqueue_emit(dart_handle* h, const dart_tree_out* o, cudaStream_t st) {
    const EmitArgs a = emit_args(h, o);
    const int pi = prof_begin(h, kEmit, st);
    const cudaError_t e = launch_prune_emit(a, st);
    prof_end(h, pi, st);
    return e == cudaSuccess ? DART_OK : DART_ERR_CUDA;
}

// The fused small-problem round: one cooperative kernel (dart_round.cu).
int enqueue_fused_round(dart_handle* h, const float* dlog, const float* anchor, const dart_tree_out* out,
                        cudaStream_t st) {
    const dart_config& c = h->cfg;
    if (h->f_dirty) return DART_ERR_STATE;  // dart_status_sync first (it resets the barrier)
    RoundArgs a;
    std::memset(&a, 0, sizeof a);
    a.V = c.V;
    a.d = c.d;
    a.L = c.L;
    a.W = c.W;
    a.k = c.k;
    a.nseq = c.nseq;
    a.G = h->fused_G;
    a.R = h->fused_R;
    a.ecache = h->fused_ecache ? 1 : 0;
    a.mstage = h->fused_mstage ? 1 : 0;
    a.stage_bytes = h->fused_stage;
    a.wres = h->fused_wres ? 1 : 0;
    for (int i = 0; i <= c.L; i++) a.caps[i] = h->caps[i];
    a.beta = c.beta;
    a.invT = c.temperature > 0.0f ? 1.0f / c.temperature : 1.0f;
    a.eps = c.rms_eps;
    a.E = static_cast<const float*>(h->E);
    a.Wi = static_cast<const float*>(h->Wi);
    a.Wo = static_cast<const float*>(h->Wo);
    a.dlog = dlog;
    a.anchor = anchor;
    a.h0 = h->hbuf[0];
    a.h1 = h->hbuf[1];
    a.rbuf = h->f_rbuf;
    a.abuf = h->f_abuf;
    a.ssqp = h->f_ssqp;
    a.pms = h->f_pms;
    a.pkey = h->f_pkey;
    a.node_logq = h->node_logq;
    a.node_lse = h->node_lse;
    a.node_tok = h->node_tok;
    a.tree_tok = h->tree_tok;
    a.tree_parent = h->tree_parent;
    a.tree_count = h->tree_count;
    a.tree_score = h->tree_score;
    a.child_prow = h->child_prow;
    a.child_tok = h->child_tok;
    a.status = h->status;
    a.bar = h->f_bar;
    a.abort = h->f_abort;
    a.emit = emit_args(h, out);
    const int pi = prof_begin(h, kFusedRound, st);
    const cudaError_t e = h->fused_cluster ? launch_round_cluster_f32(a, h->fused_nm, h->fused_smem, st)
                                           : launch_round_small_f32(a, h->fused_nm, h->fused_smem, st);
    prof_end(h, pi, st);
    h->cur = (c.L - 1) & 1;  // depth L's states: the parity buffer of depth L
    h->next_depth = c.L + 1;
    return e == cudaSuccess ? DART_OK : DART_ERR_CUDA;
}

int enqueue_round(dart_handle* h, const float* dlog, const float* anchor, const dart_tree_out* out, cudaStream_t st) {
    if (h->fused) return enqueue_fused_round(h, dlog, anchor, out, st);
    for (int dep = 1; dep <= h->cfg.L; dep++) {
        int rc = enqueue_depth(h, h->cfg, h->plans, dep, dlog, anchor, st);
        if (rc != DART_OK) return rc;
    }
    h->next_depth = h->cfg.L + 1;
    return enqueue_emit(h, out, st);
}

// Domino-chain + DDTree (Table 2): the chain is Algorithm 1 with W = k = 1
// (one node per sequence and depth: its argmax child continues the chain),
// which also keeps every depth's scaled logits and log-sum-exp; then the
// chain's best Bp = min(B, V) children of every depth, best first, and
// DDTree's best-first search over those position-wise distributions.
int enqueue_chain_ddtree(dart_handle* h, const float* dlog, const float* anchor, const dart_tree_out* out,
                         cudaStream_t st) {
    const dart_config& c = h->cfg;
    for (int dep = 1; dep <= c.L; dep++) {
        DepthOutputs o;
        o.zout = h->zrows + static_cast<size_t>(dep - 1) * c.V;
        o.zout_stride = static_cast<long long>(c.L) * c.V;
        o.lse_hist = h->chain_lse + (dep - 1);
        o.lse_hist_stride = c.L;
        const int rc = enqueue_depth(h, h->ccfg, h->cplans, dep, dlog, anchor, st, &o);
        if (rc != DART_OK) return rc;
    }
    int pi = prof_begin(h, kRowTopk, st);
    cudaError_t e = launch_row_topk_by_value(h->zrows, c.nseq * c.L, c.V, h->Bp, h->ddt_S, h->ddt_tok, h->ddt_z,
                                             h->Bp, h->ddt_part, h->ddt_ticket, st);
    prof_end(h, pi, st);
    if (e != cudaSuccess) return DART_ERR_CUDA;
    DdtArgs a;
    std::memset(&a, 0, sizeof a);
    a.L = c.L;
    a.B = c.B;
    a.Bp = h->Bp;
    a.nseq = c.nseq;
    a.pos_offset = c.pos_offset;
    a.beta = c.beta;
    a.tok = h->ddt_tok;
    a.zval = h->ddt_z;
    a.lse = h->chain_lse;
    a.tokens = out->tokens;
    a.parents = out->parents;
    a.depths = out->depths;
    a.pos_ids = out->pos_ids;
    a.n_nodes = out->n_nodes;
    a.scores = out->scores;
    a.mask = out->mask;
    a.status = h->status;
    pi = prof_begin(h, kDdtree, st);
    e = launch_ddtree(a, st);
    prof_end(h, pi, st);
    return e == cudaSuccess ? DART_OK : DART_ERR_CUDA;
}

// Sequential correction with heap (Sec. 4.1, Table 2): B pops, each
// correcting the popped prefix before the next: its state (head update of
// one node per sequence) and its children over the vocabulary (LM-head,
// merge for the log-sum-exp, the best Bp children best first).  The last pop
// needs no correction, nor does any pop when L = 1.
int enqueue_seq_heap(dart_handle* h, const float* dlog, const float* anchor, const dart_tree_out* out,
                     cudaStream_t st) {
    const dart_config& c = h->cfg;
    const dart_config& cc = h->ccfg;
    const DepthPlan& p = h->cplans[1];  // one node per sequence
    const bool tc = h->wdtype == DART_BF16;
    const size_t S1 = static_cast<size_t>(c.B) + 1;
    SeqHeapArgs a;
    std::memset(&a, 0, sizeof a);
    a.L = c.L;
    a.B = c.B;
    a.Bp = h->Bp;
    a.nseq = c.nseq;
    a.d = c.d;
    a.pos_offset = c.pos_offset;
    a.bhalf = kNPadMax;
    a.beta = c.beta;
    a.anchor = anchor;
    a.tab = h->sh_tab;
    a.ltok = h->sh_ltok;
    a.lz = h->sh_lz;
    a.llse = h->sh_llse;
    a.next = h->sh_next;
    a.offer = h->sh_offer;
    a.npop = h->sh_npop;
    a.hin = h->hbuf[0];
    a.HL = tc ? h->HL : nullptr;
    a.hout = h->hbuf[1];
    a.child_prow = h->child_prow;
    a.child_tok = h->child_tok;
    a.dlog_row = h->sh_dlog_row;
    a.tokens = out->tokens;
    a.parents = out->parents;
    a.depths = out->depths;
    a.pos_ids = out->pos_ids;
    a.n_nodes = out->n_nodes;
    a.scores = out->scores;
    a.mask = out->mask;
    a.status = h->status;
    // scoring of one node per sequence, its best Bp children into slot `slot`
    auto score = [&](int slot, const float* h32, const int* dlog_row, bool first) -> int {
        LmheadArgs la = lmhead_args(h, cc, p, dlog, h32);
        la.dlog_row = dlog_row;  // null: position 0 (the root's children)
        la.gthr = first ? h->gthr : nullptr;
        la.zout = h->sh_zrow;
        la.zout_stride = c.V;
        int pi = prof_begin(h, kLmhead, st);
        cudaError_t e = tc ? launch_lmhead_tc(&h->tmE, &h->tmH[ng_index(p.NG)], la, p.smem, st) : launch_lmhead_f32(la, st);
        prof_end(h, pi, st);
        if (e != cudaSuccess) return DART_ERR_CUDA;
        SelectArgs sa = select_args(h, cc, p, 1);
        sa.gthr = la.gthr;
        sa.lse_hist = h->sh_llse + slot;
        sa.lse_hist_stride = static_cast<long long>(S1);
        pi = prof_begin(h, kSelect, st);
        e = launch_merge_select(sa, st);
        prof_end(h, pi, st);
        if (e != cudaSuccess) return DART_ERR_CUDA;
        pi = prof_begin(h, kRowTopk, st);
        e = launch_row_topk_by_value(h->sh_zrow, c.nseq, c.V, h->Bp, h->sh_S, h->sh_ltok + slot * h->Bp,
                                     h->sh_lz + slot * h->Bp, static_cast<long long>(S1) * h->Bp, h->sh_part,
                                     h->sh_ticket, st);
        prof_end(h, pi, st);
        return e == cudaSuccess ? DART_OK : DART_ERR_CUDA;
    };
    int pi = prof_begin(h, kPrep, st);
    cudaError_t e = launch_prep_anchor(anchor, c.nseq, c.d, h->hbuf[0], tc ? h->HL : nullptr, kNPadMax, h->gthr,
                                       kNPadMax, st);
    prof_end(h, pi, st);
    if (e != cudaSuccess) return DART_ERR_CUDA;
    int rc = score(0, h->hbuf[0], nullptr, true);
    if (rc != DART_OK) return rc;
    for (int t = 0; t < c.B; t++) {
        pi = prof_begin(h, kSeqStep, st);
        e = launch_seqheap_step(a, t, st);
        prof_end(h, pi, st);
        if (e != cudaSuccess) return DART_ERR_CUDA;
        if (c.L == 1 || t + 1 == c.B) continue;
        rc = enqueue_head_update(h, cc, p, h->hbuf[0], h->hbuf[1], false, st);
        if (rc == DART_OK) rc = score(t + 1, h->hbuf[1], h->sh_dlog_row, false);
        if (rc != DART_OK) return rc;
    }
    pi = prof_begin(h, kSeqEmit, st);
    e = launch_seqheap_emit(a, st);
    prof_end(h, pi, st);
    return e == cudaSuccess ? DART_OK : DART_ERR_CUDA;
}

int check_inputs(const dart_handle* h, const float* dlog, const float* anchor, bool need_anchor) {
    if (!dlog || !aligned4(dlog)) return DART_ERR_INVALID;
    if (need_anchor && (!anchor || !aligned16(anchor))) return DART_ERR_INVALID;  // read with 16-byte loads
    (void)h;
    return DART_OK;
}

// Keeps `ge` in the handle's graph cache, destroying the least recently used
// entry when the cache is full (a graph launched earlier on the caller's
// stream may still run: cudaGraphExecDestroy defers its release until then),
// and launches it.
cudaError_t cache_and_launch(dart_handle* h, const GraphEntry& ge, cudaStream_t st) {
    if (h->graphs.size() >= kMaxGraphs) {
        size_t lru = 0;
        for (size_t i = 1; i < h->graphs.size(); i++)
            if (h->graphs[i].last_use < h->graphs[lru].last_use) lru = i;
        cudaGraphExecDestroy(h->graphs[lru].exec);
        h->graphs.erase(h->graphs.begin() + static_cast<long>(lru));
    }
    h->graphs.push_back(ge);
    return cudaGraphLaunch(ge.exec, st);
}

int enqueue_kind(dart_handle* h, int kind, const float* dlog, const float* anchor, const dart_tree_out* out,
                 cudaStream_t st) {
    switch (kind) {
        case kRoundChainDdtree: return enqueue_chain_ddtree(h, dlog, anchor, out, st);
        case kRoundSeqHeap: return enqueue_seq_heap(h, dlog, anchor, out, st);
        default: return enqueue_round(h, dlog, anchor, out, st);
    }
}

// After a round of `kind`: the state the test hooks see.  Algorithm 1's
// rounds leave every depth readable; the best-first constructions leave no
// Algorithm 1 frontier (dart_get_chain reads the chain).
void finish_round(dart_handle* h, int kind, bool ok) {
    h->last_kind = kind;
    if (!ok) {
        h->next_depth = 1;
        return;
    }
    h->next_depth = h->cfg.L + 1;
    if (kind == kRoundDartree) h->last_rows = h->plans[h->cfg.L].N;
}

// One round of construction `kind`: launched as one cached CUDA graph per
// distinct (kind, inputs, outputs) set, or enqueued directly when profiling
// or when the caller is capturing the stream.
int run_round(dart_handle* h, int kind, const float* dlog, const float* anchor, const dart_tree_out* out,
              void* stream) {
    if (!h) return DART_ERR_INVALID;
    int rc = check_inputs(h, dlog, anchor, true);
    if (rc == DART_OK) rc = check_out(out);
    if (rc != DART_OK) return rc;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(st, &cs) != cudaSuccess) return DART_ERR_CUDA;
    // (the fused round is one launch already: no graph)
    if (h->profiling || cs != cudaStreamCaptureStatusNone || (kind == kRoundDartree && h->fused)) {
        rc = enqueue_kind(h, kind, dlog, anchor, out, st);
        finish_round(h, kind, rc == DART_OK);
        return rc;
    }
    const void* key[10] = {reinterpret_cast<const void*>(static_cast<uintptr_t>(kind)),
                           dlog, anchor, out->tokens, out->parents, out->depths,
                           out->pos_ids, out->scores, out->n_nodes, out->mask};
    for (auto& g : h->graphs) {
        if (std::memcmp(g.key, key, sizeof key) == 0) {
            finish_round(h, kind, true);
            g.last_use = ++h->graph_clock;
            return cuda_err(cudaGraphLaunch(g.exec, st));
        }
    }
    cudaGraph_t graph = nullptr;
    if (cudaStreamBeginCapture(h->cap_stream, cudaStreamCaptureModeThreadLocal) != cudaSuccess) return DART_ERR_CUDA;
    rc = enqueue_kind(h, kind, dlog, anchor, out, h->cap_stream);
    cudaError_t ce = cudaStreamEndCapture(h->cap_stream, &graph);
    if (rc != DART_OK || ce != cudaSuccess) {
        if (graph) cudaGraphDestroy(graph);
        finish_round(h, kind, false);
        return rc != DART_OK ? rc : DART_ERR_CUDA;
    }
    GraphEntry ge;
    std::memcpy(ge.key, key, sizeof key);
    ce = cudaGraphInstantiate(&ge.exec, graph, 0);
    cudaGraphDestroy(graph);
    if (ce != cudaSuccess) {
        finish_round(h, kind, false);
        return DART_ERR_CUDA;
    }
    ge.last_use = ++h->graph_clock;
    finish_round(h, kind, true);
    return cuda_err(cache_and_launch(h, ge, st));
}

}  // namespace

extern "C" {

int dart_version(void) { return kVersion; }

const char* dart_status_string(int code) {
    switch (code) {
        case DART_OK: return "ok";
        case DART_ERR_INVALID: return "invalid argument";
        case DART_ERR_CUDA: return "CUDA error";
        case DART_ERR_NOMEM: return "out of memory";
        case DART_ERR_TIMEOUT: return "device wait timed out";
        case DART_ERR_STATE: return "call out of order";
        case DART_ERR_UNSUPPORTED: return "unsupported device or configuration";
        case DART_ERR_BOUNDS: return "device index check failed (debug build)";
        default: return "unknown status";
    }
}

int dart_init_head(dart_handle** out, const dart_config* cfg, int wdtype, const void* W_i, const void* W_o,
                   const void* E, void* stream) {
    if (!out) return DART_ERR_INVALID;
    *out = nullptr;
    int rc = validate_cfg(cfg);
    if (rc != DART_OK) return rc;
    if (wdtype != DART_F32 && wdtype != DART_BF16) return DART_ERR_INVALID;
    if (!W_i || !W_o || !E || !aligned16(W_i) || !aligned16(W_o) || !aligned16(E)) return DART_ERR_INVALID;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return DART_ERR_CUDA;
    int major = 0, minor = 0, sms = 0, optin = 0, l2 = 0;
    if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&l2, cudaDevAttrL2CacheSize, dev) != cudaSuccess)
        return DART_ERR_CUDA;
    if (major != 10 || minor != 3) return DART_ERR_UNSUPPORTED;  // built for sm_103a only
    dart_handle* h = new (std::nothrow) dart_handle();
    if (!h) return DART_ERR_NOMEM;
    h->cfg = *cfg;
    h->wdtype = wdtype;
    h->Wi = W_i;
    h->Wo = W_o;
    h->E = E;
    h->dev = dev;
    h->num_sms = sms;
    h->smem_optin = optin;
    h->l2_bytes = l2;
    h->next_depth = 1;
    if (wdtype == DART_BF16 && tc_set_smem_limits(optin) != cudaSuccess) rc = DART_ERR_CUDA;
    {
        // AUTO: the tiled copy of E where it was measured faster per round on
        // GB300 (A/B, same process): d <= 3072 with at most 16 nodes per
        // depth (Qwen3-4B shape -2 to -4 %, sweep W = 8); elsewhere the gain
        // was within +-1 % (d = 4096 with 16 nodes, 8 x 32 nodes, 64 nodes)
        // or a loss (+3.7 % with 32 nodes at d = 2560)
        int max_nodes = 0, width = 1;
        for (int dep = 1; dep <= cfg->L; dep++) {
            max_nodes = std::max(max_nodes, cfg->nseq * width);
            width = std::min(cfg->W, width * cfg->k);
        }
        const bool auto_on = cfg->d <= 3072 && max_nodes <= 16;
        h->tiled = wdtype == DART_BF16 &&
                   (cfg->weights_tiled == DART_ON || (cfg->weights_tiled == DART_AUTO && auto_on));
    }
    h->wtiled = wdtype == DART_BF16 && cfg->head_weights_tiled == DART_ON;
    h->Kwi = (wdtype == DART_BF16 && cfg->head_split != DART_OFF) ? cfg->d : 2 * cfg->d;
    if (rc == DART_OK) rc = build_plans(h, h->cfg, h->caps, h->plans);
    if (rc == DART_OK) rc = plan_fused_round(h);
    if (rc == DART_OK && cfg->variants) {
        // the best-first constructions score one node per sequence at a time
        // over the full vocabulary and keep its best min(B, V) children
        if (cfg->cand_k != 0 || cfg->nseq > 64) rc = DART_ERR_UNSUPPORTED;
        h->ccfg = *cfg;
        h->ccfg.W = 1;
        h->ccfg.k = 1;
        h->Bp = std::min(cfg->B, cfg->V);
        h->ddt_S = cand_topk_slices(cfg->V, h->Bp, cfg->nseq * cfg->L, sms);
        h->sh_S = cand_topk_slices(cfg->V, h->Bp, cfg->nseq, sms);
        if (rc == DART_OK) rc = build_plans(h, h->ccfg, h->ccaps, h->cplans);
        if (rc == DART_OK && (cfg->variants & DART_VARIANT_CHAIN_DDTREE) &&
            ddtree_smem(cfg->L, h->Bp, cfg->B) > optin)
            rc = DART_ERR_UNSUPPORTED;
    }
    if (rc == DART_OK) rc = alloc_workspace(h);
    if (rc == DART_OK && wdtype == DART_BF16) rc = make_tensor_maps(h);
    if (rc == DART_OK && h->Qtab) rc = compute_qtab(h, static_cast<cudaStream_t>(stream));
    if (rc == DART_OK && (h->tiled || h->wtiled)) {
        cudaStream_t st0 = static_cast<cudaStream_t>(stream);
        const __nv_bfloat16* wi = static_cast<const __nv_bfloat16*>(W_i);
        cudaError_t e = cudaSuccess;
        if (h->tiled) e = launch_retile(static_cast<const __nv_bfloat16*>(E), cfg->V, cfg->d, cfg->d, h->Et, st0);
        if (h->wtiled && e == cudaSuccess) e = launch_retile(wi, cfg->d, h->Kwi, 2ll * cfg->d, h->Wit, st0);
        if (h->wtiled && e == cudaSuccess)
            e = launch_retile(static_cast<const __nv_bfloat16*>(W_o), cfg->d, cfg->d, cfg->d, h->Wot, st0);
        rc = cuda_err(e);
    }
    if (rc == DART_OK && cudaStreamCreateWithFlags(&h->cap_stream, cudaStreamNonBlocking) != cudaSuccess)
        rc = DART_ERR_CUDA;
    if (rc == DART_OK && h->Qtab &&
        (cudaStreamCreateWithFlags(&h->side, cudaStreamNonBlocking) != cudaSuccess ||
         cudaEventCreateWithFlags(&h->ev_fork, cudaEventDisableTiming) != cudaSuccess ||
         cudaEventCreateWithFlags(&h->ev_join, cudaEventDisableTiming) != cudaSuccess))
        rc = DART_ERR_CUDA;
    if (rc == DART_OK && cudaDeviceSynchronize() != cudaSuccess) rc = DART_ERR_CUDA;
    if (rc == DART_OK && h->Qtab) {
        // the table's GEMM waits with a time limit: one that gave up left Q incomplete
        int word = 0;
        if (cudaMemcpy(&word, h->status, sizeof word, cudaMemcpyDeviceToHost) != cudaSuccess)
            rc = DART_ERR_CUDA;
        else if (word & kDevTimeout)
            rc = DART_ERR_TIMEOUT;
    }
    if (rc != DART_OK) {
        release(h);
        delete h;
        return rc;
    }
    *out = h;
    return DART_OK;
}

int dart_expand_depth(dart_handle* h, int depth, const float* drafter_logits, const float* anchor_h, void* stream) {
    if (!h) return DART_ERR_INVALID;
    if (depth < 1 || depth > h->cfg.L) return DART_ERR_INVALID;
    int rc = check_inputs(h, drafter_logits, anchor_h, depth == 1);
    if (rc != DART_OK) return rc;
    if (depth != 1 && (depth != h->next_depth || h->last_kind != kRoundDartree)) return DART_ERR_STATE;
    rc = enqueue_depth(h, h->cfg, h->plans, depth, drafter_logits, anchor_h, static_cast<cudaStream_t>(stream));
    h->next_depth = rc == DART_OK ? depth + 1 : 1;
    h->last_kind = kRoundDartree;
    return rc;
}

int dart_prune_and_emit(dart_handle* h, const dart_tree_out* out, void* stream) {
    if (!h) return DART_ERR_INVALID;
    int rc = check_out(out);
    if (rc != DART_OK) return rc;
    if (h->next_depth != h->cfg.L + 1 || h->last_kind != kRoundDartree) return DART_ERR_STATE;
    return enqueue_emit(h, out, static_cast<cudaStream_t>(stream));
}

int dart_build_tree(dart_handle* h, const float* drafter_logits, const float* anchor_h, const dart_tree_out* out,
                    void* stream) {
    return run_round(h, kRoundDartree, drafter_logits, anchor_h, out, stream);
}

int dart_build_tree_fixed(dart_handle* h, const float* drafter_logits, const float* anchor_h,
                          const dart_tree_out* out, void* stream) {
    if (!h) return DART_ERR_INVALID;
    int total = 0;
    for (int dep = 1; dep <= h->cfg.L; dep++) total += h->caps[dep];
    if (h->cfg.B < total) return DART_ERR_INVALID;  // every retained node must fit: no pruning
    return run_round(h, kRoundDartree, drafter_logits, anchor_h, out, stream);
}

int dart_build_chain_ddtree(dart_handle* h, const float* drafter_logits, const float* anchor_h,
                            const dart_tree_out* out, void* stream) {
    if (!h) return DART_ERR_INVALID;
    if (!(h->cfg.variants & DART_VARIANT_CHAIN_DDTREE)) return DART_ERR_STATE;
    return run_round(h, kRoundChainDdtree, drafter_logits, anchor_h, out, stream);
}

int dart_build_seq_heap(dart_handle* h, const float* drafter_logits, const float* anchor_h, const dart_tree_out* out,
                        void* stream) {
    if (!h) return DART_ERR_INVALID;
    if (!(h->cfg.variants & DART_VARIANT_SEQ_HEAP)) return DART_ERR_STATE;
    return run_round(h, kRoundSeqHeap, drafter_logits, anchor_h, out, stream);
}

int dart_get_chain(dart_handle* h, int32_t* tok, float* lse, void* stream) {
    if (!h) return DART_ERR_INVALID;
    if (h->last_kind != kRoundChainDdtree || h->next_depth != h->cfg.L + 1) return DART_ERR_STATE;
    const size_t n = static_cast<size_t>(h->cfg.nseq) * h->cfg.L;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    cudaError_t e = cudaSuccess;
    // the chain ran with W = 1: its depth-d node of sequence s is tree slot s * L + d - 1
    if (tok) e = cudaMemcpyAsync(tok, h->tree_tok, n * 4, cudaMemcpyDeviceToDevice, st);
    if (lse && e == cudaSuccess) e = cudaMemcpyAsync(lse, h->chain_lse, n * 4, cudaMemcpyDeviceToDevice, st);
    return cuda_err(e);
}

int dart_build_tree_host(dart_handle* h, const float* drafter_logits_host, const float* anchor_host,
                         const dart_tree_out* out_host, void* stream) {
    if (!h || !drafter_logits_host || !anchor_host) return DART_ERR_INVALID;
    int rc = check_out(out_host);
    if (rc != DART_OK) return rc;
    const dart_config& c = h->cfg;
    const size_t n_dlog = static_cast<size_t>(c.nseq) * c.L * c.V;
    const size_t n_anchor = static_cast<size_t>(c.nseq) * c.d;
    const size_t nB = static_cast<size_t>(c.nseq) * c.B;
    const size_t nmask = nB * ((c.B + 63) / 64);
    if (!h->staged) {
        rc = dalloc(h, &h->st_dlog, n_dlog);
        if (rc == DART_OK) rc = dalloc(h, &h->st_anchor, n_anchor);
        if (rc == DART_OK) rc = dalloc(h, &h->st_out.tokens, nB);
        if (rc == DART_OK) rc = dalloc(h, &h->st_out.parents, nB);
        if (rc == DART_OK) rc = dalloc(h, &h->st_out.depths, nB);
        if (rc == DART_OK) rc = dalloc(h, &h->st_out.pos_ids, nB);
        if (rc == DART_OK) rc = dalloc(h, &h->st_out.scores, nB);
        if (rc == DART_OK) rc = dalloc(h, &h->st_out.n_nodes, static_cast<size_t>(c.nseq));
        if (rc == DART_OK) rc = dalloc(h, &h->st_out.mask, nmask);
        if (rc != DART_OK) return rc;
        h->staged = true;
    }
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (cudaMemcpyAsync(h->st_dlog, drafter_logits_host, n_dlog * 4, cudaMemcpyHostToDevice, st) != cudaSuccess ||
        cudaMemcpyAsync(h->st_anchor, anchor_host, n_anchor * 4, cudaMemcpyHostToDevice, st) != cudaSuccess)
        return DART_ERR_CUDA;
    rc = dart_build_tree(h, h->st_dlog, h->st_anchor, &h->st_out, stream);
    if (rc != DART_OK) return rc;
    const dart_tree_out& d = h->st_out;
    const dart_tree_out& o = *out_host;
    cudaError_t e = cudaSuccess;
    e = cudaMemcpyAsync(o.tokens, d.tokens, nB * 4, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaMemcpyAsync(o.parents, d.parents, nB * 4, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaMemcpyAsync(o.depths, d.depths, nB * 4, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaMemcpyAsync(o.pos_ids, d.pos_ids, nB * 4, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaMemcpyAsync(o.scores, d.scores, nB * 4, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaMemcpyAsync(o.n_nodes, d.n_nodes, c.nseq * 4, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaMemcpyAsync(o.mask, d.mask, nmask * 8, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    return cuda_err(e);
}

int dart_get_frontier(dart_handle* h, int depth, int32_t* tok, int32_t* parent_slot, float* score, int32_t* count,
                      void* stream) {
    if (!h || depth < 1 || depth > h->cfg.L) return DART_ERR_INVALID;
    if (depth >= h->next_depth || h->last_kind != kRoundDartree) return DART_ERR_STATE;
    const dart_config& c = h->cfg;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const size_t W = c.W;
    cudaError_t e = cudaSuccess;
    for (int s = 0; s < c.nseq && e == cudaSuccess; s++) {
        const size_t src = (static_cast<size_t>(s) * c.L + depth - 1) * W;
        if (tok) e = cudaMemcpyAsync(tok + s * W, h->tree_tok + src, W * 4, cudaMemcpyDeviceToDevice, st);
        if (parent_slot && e == cudaSuccess)
            e = cudaMemcpyAsync(parent_slot + s * W, h->tree_parent + src, W * 4, cudaMemcpyDeviceToDevice, st);
        if (score && e == cudaSuccess)
            e = cudaMemcpyAsync(score + s * W, h->tree_score + src, W * 4, cudaMemcpyDeviceToDevice, st);
        if (count && e == cudaSuccess)
            e = cudaMemcpyAsync(count + s, h->tree_count + s * c.L + depth - 1, 4, cudaMemcpyDeviceToDevice, st);
    }
    return cuda_err(e);
}

int dart_get_node_topk(dart_handle* h, int32_t* tok, float* logq, float* lse, int* rows, void* stream) {
    if (!h) return DART_ERR_INVALID;
    if (h->next_depth < 2 || h->last_kind != kRoundDartree) return DART_ERR_STATE;
    const int dep = h->next_depth - 1;
    const int N = h->plans[dep].N;
    if (rows) *rows = N;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const size_t nk = static_cast<size_t>(N) * h->cfg.k;
    cudaError_t e = cudaSuccess;
    if (tok) e = cudaMemcpyAsync(tok, h->node_tok, nk * 4, cudaMemcpyDeviceToDevice, st);
    if (logq && e == cudaSuccess) e = cudaMemcpyAsync(logq, h->node_logq, nk * 4, cudaMemcpyDeviceToDevice, st);
    if (lse && e == cudaSuccess) e = cudaMemcpyAsync(lse, h->node_lse, N * 4, cudaMemcpyDeviceToDevice, st);
    return cuda_err(e);
}

int dart_get_states(dart_handle* h, float* states, int* rows, void* stream) {
    if (!h) return DART_ERR_INVALID;
    if (h->next_depth < 2 || h->last_kind != kRoundDartree) return DART_ERR_STATE;
    const int dep = h->next_depth - 1;
    const int R = dep < h->cfg.L ? h->plans[dep].Nc : h->plans[dep].N;
    if (rows) *rows = R;
    if (!states) return DART_OK;
    return cuda_err(cudaMemcpyAsync(states, h->hbuf[h->cur], static_cast<size_t>(R) * h->cfg.d * 4,
                                    cudaMemcpyDeviceToDevice, static_cast<cudaStream_t>(stream)));
}

int dart_status_sync(dart_handle* h, void* stream) {
    if (!h) return DART_ERR_INVALID;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    int word = 0;
    if (cudaStreamSynchronize(st) != cudaSuccess) return DART_ERR_CUDA;
    if (cudaMemcpy(&word, h->status, sizeof word, cudaMemcpyDeviceToHost) != cudaSuccess) return DART_ERR_CUDA;
    if (cudaMemset(h->status, 0, sizeof word) != cudaSuccess) return DART_ERR_CUDA;
    if (word & kDevTimeout) {
        // a fused round that gave up left its grid barrier mid-way
        if (h->f_bar && (cudaMemset(h->f_bar, 0, kRoundBarWords * sizeof(unsigned)) != cudaSuccess ||
                         cudaMemset(h->f_abort, 0, sizeof(int)) != cudaSuccess))
            return DART_ERR_CUDA;
        h->f_dirty = false;
        return DART_ERR_TIMEOUT;
    }
    if (word & kDevBounds) return DART_ERR_BOUNDS;
    if (word & kDevOrphan) return DART_ERR_STATE;
    return DART_OK;
}

int dart_debug_build(void) { return debug_build() ? 1 : 0; }

int dart_test_barrier_timeout(dart_handle* h, int limit_us, void* stream) {
    if (!h || limit_us < 1 || limit_us > 2000000) return DART_ERR_INVALID;
    if (!h->fused) return DART_ERR_STATE;
    h->f_dirty = true;
    return cuda_err(launch_barrier_probe(h->f_bar, h->f_abort, h->status,
                                         static_cast<unsigned long long>(limit_us) * 1000ull,
                                         static_cast<cudaStream_t>(stream)));
}

int dart_test_bounds_report(dart_handle* h, void* stream) {
    if (!h) return DART_ERR_INVALID;
    return cuda_err(launch_bounds_probe(h->status, static_cast<cudaStream_t>(stream)));
}

int dart_test_wait_timeout(dart_handle* h, int limit_us, int64_t* elapsed_ns, void* stream) {
    if (!h || limit_us < 1 || limit_us > 2000000) return DART_ERR_INVALID;
    if (elapsed_ns && (reinterpret_cast<uintptr_t>(elapsed_ns) & 7u)) return DART_ERR_INVALID;
    return cuda_err(launch_wait_probe(h->status, static_cast<unsigned long long>(limit_us) * 1000ull,
                                      reinterpret_cast<long long*>(elapsed_ns), static_cast<cudaStream_t>(stream)));
}

int dart_set_profiling(dart_handle* h, int enable) {
    if (!h) return DART_ERR_INVALID;
    h->profiling = enable != 0;
    h->ev_used = 0;
    return DART_OK;
}

int dart_profile_read_kinds(dart_handle* h, float* ms, int* launches, int nkinds) {
    if (!h || nkinds < 0 || nkinds > kNumKinds) return DART_ERR_INVALID;
    float tot[kNumKinds] = {0};
    int cnt[kNumKinds] = {0};
    const int pairs = h->ev_used / 2;
    if (pairs > 0 && cudaEventSynchronize(h->ev[h->ev_used - 1]) != cudaSuccess) return DART_ERR_CUDA;
    for (int i = 0; i < pairs; i++) {
        float t = 0.0f;
        if (cudaEventElapsedTime(&t, h->ev[2 * i], h->ev[2 * i + 1]) != cudaSuccess) return DART_ERR_CUDA;
        const int k = h->ev_kind[2 * i];
        if (k >= 0 && k < kNumKinds) {
            tot[k] += t;
            cnt[k]++;
        }
    }
    for (int k = 0; k < nkinds; k++) {
        if (ms) ms[k] = tot[k];
        if (launches) launches[k] = cnt[k];
    }
    h->ev_used = 0;
    return DART_OK;
}

int dart_profile_read(dart_handle* h, float* lmhead_ms, int* lmhead_launches) {
    return dart_profile_read_kinds(h, lmhead_ms, lmhead_launches, 1);
}

int dart_launches_per_round(dart_handle* h) {
    if (!h) return DART_ERR_INVALID;
    const int L = h->cfg.L;
    if (h->fused) return 1;
    // prep, (LM-head + select) per depth, then per depth but the last:
    // gather, W_i GEMM, [SiLU,] W_o GEMM, residual-norm; or with the split
    // first layer: W_i[:, 0:d] GEMM, gather + SiLU, W_o GEMM, residual-norm,
    // and beside them the early prefetch of the next depth's E tiles; or
    // (fp32, d <= 1024) the whole update in one launch; prune-emit
    const bool tc = h->wdtype == DART_BF16;
    int n = 1 + 2 * L + 1 + (h->cfg.cand_k > 0 ? 1 : 0);
    for (int dep = 1; dep <= L; dep++) n += h->plans[dep].bound > 0 ? 1 : 0;
    for (int dep = 1; dep < L; dep++) {
        const DepthPlan& p = h->plans[dep];
        if (!tc && head_small_f32_slices(h->cfg.d) > 0) {
            n += 1;
            continue;
        }
        n += (p.split || (tc && p.g1.mode != kGemmPartials)) ? 4 : 5;
        if (p.side && h->cfg.cand_k == 0 && h->plans[dep + 1].epf > 0) n += 1;
    }
    return n;
}

void dart_destroy(dart_handle* h) {
    if (!h) return;
    cudaDeviceSynchronize();
    release(h);
    delete h;
}

}  // extern "C"
