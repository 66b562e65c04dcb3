// Internal launch interface between the C-ABI layer and the kernels.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace dart {

// cuTensorMapEncodeTiled from the driver (NULL if unavailable), looked up once.
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn tensor_map_encoder();

// Raises `fn`'s dynamic shared-memory limit to the most the device allows
// beside the kernel's static shared memory.  Kernel attributes are
// process-wide: a handle never lowers a limit another handle's plan needs.
inline cudaError_t set_max_dynamic_smem(const void* fn) {
    int dev = 0, optin = 0;
    cudaFuncAttributes fa;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    if (e == cudaSuccess) e = cudaFuncGetAttributes(&fa, fn);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 optin - static_cast<int>(fa.sharedSizeBytes));
    return e;
}

// Launches `kernel` with programmatic stream serialization (PDL), so its
// prologue can overlap the tail of the previous kernel in the stream.
bool pdl_enabled();

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                       Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl_enabled() ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
}

// The same with thread-block clusters of `cluster_x` consecutive CTAs.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl_cluster(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                               int cluster_x, Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = static_cast<unsigned>(cluster_x);
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl_enabled() ? 2 : 1;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
}

// LM-head scoring (Algorithm 1: correct every prefix of S_{d-1} over the full
// vocabulary, Appendix D "Full"): per node n and vocabulary row v,
//   z[n][v] = (Dlog[seq(n)][dep-1][v] + E[v] . h[n]) * invT,
// reduced on chip to per-CTA (max, sum exp) and top-k keys.
struct LmheadArgs {
    int V, d, N;          // vocabulary, hidden, nodes at this depth
    int NG, G;            // nodes per group (multiple of 16), groups
    int nV;               // vocabulary ranges (CTAs per group)
    int k;
    int tiles;            // ceil(V / 128)
    int P;                // nodes per sequence (node n belongs to sequence n / P)
    float invT;
    const float* dlog;    // [nseq][L][V]
    long long dlog_seq_stride;  // L * V
    long long dlog_row_off;     // (dep-1) * V
    int bhalf;            // row offset of the lo half in the bf16 state operand
    int stages;           // smem pipeline depth (tcgen05 kernel)
    int l2pf;             // A tiles prefetched into L2 before the wait on the previous kernel
    float2* part_ms;      // [nV][N]
    uint64_t* part_key;   // [nV][N][k]
    int* status;
    const float* h32;     // fp32 states [N][d] (fp32 kernel)
    const float* E32;     // fp32 table [V][d]   (fp32 kernel)
    uint64_t* gthr;       // [N] cross-CTA top-k bounds, zero before the launch (may be null)
    int e_tiled;          // the E tensor map is over the tiled copy (launch_retile), not [V][d]
    int DS;               // fp32 kernel: blocks (one cluster) sharing a vocabulary range, each a slice of d
    // optional (null: unused)
    const int* dlog_row;  // [nseq] drafter row of each sequence's nodes (replaces dlog_row_off / V)
    float* zout;          // z[n][v] written to zout[n * zout_stride + v] (node groups <= 64)
    long long zout_stride;
    const float* seed_y;  // [N][seed_R] seed scores (launch_seed_score): the filter starts from each
    int seed_R;           // node's k-th largest, which is also published into gthr (null: no seed pass)
};

// Skinny split-K GEMM for the correction head: out[split][n][m] =
// sum_{k in split} A[m][k] * B[n][k], B given as hi + lo bf16 halves.
struct GemmArgs {
    int M, K, N;          // output features, reduction length, nodes
    int NG, G, MT, S;     // node group, groups, m tiles, k splits
    int KB;               // K / 64
    int lo_kb_end;        // k-blocks >= this have a zero lo half (skipped)
    int bhalf;
    int stages;
    int mode;             // tcgen05 path: kGemmPartials, or kGemmSiluSplit / kGemmSum (the k splits are one cluster)
    int keep_a;           // load A (the weights) evict-last: it is read again at the next depth from L2
    int a_tiled_kb;       // 0: A's tensor map is row-major [M][K]; else over a tiled copy with this many k-blocks per row of tiles
    float* out;           // fp32 path: partials [S][N][M]; kGemmSum: the sum [N][M]
    __nv_bfloat16* outL;  // kGemmSiluSplit: SiLU of the sum as hi rows [N][M], lo rows from row bhalf
    int* status;
    const float* A32;     // fp32 path: A [M][K]
    const float* B32;     // fp32 path: B [N][K]
};

constexpr int kGemmPartials = 0;   // out[split] = partial A . B^T over the split's k range
constexpr int kGemmSiluSplit = 1;  // out = split(SiLU(A . B^T)) (correction-head W_i layer)
constexpr int kGemmSum = 2;        // out = A . B^T in fp32 (correction-head W_o layer)
constexpr int kMaxClusterK = 8;    // k splits of one tile reduced on chip (portable cluster size)

// tcgen05 kernels (dart_tc.cu)
cudaError_t launch_lmhead_tc(const CUtensorMap* tmE, const CUtensorMap* tmH, const LmheadArgs& a,
                             int smem_bytes, cudaStream_t st);
cudaError_t launch_gemm_tc(const CUtensorMap* tmA, const CUtensorMap* tmB, const GemmArgs& a, int smem_bytes,
                           cudaStream_t st);
int tc_stage_bytes(int NG);
int lmhead_tc_tmem_cols(int NG);  // TMEM columns one LM-head CTA allocates
int lmhead_tc_fixed_smem(int NG, int k, int stages);
int gemm_tc_fixed_smem(int stages);
int lmhead_tc_ctas_per_sm(int NG, int smem);
int gemm_tc_ctas_per_sm(int NG, int smem);
int gemm_tc_max_clusters(int NG, int smem, int cluster);  // resident CTAs per SM (occupancy API; needs limits set)
cudaError_t tc_set_smem_limits(int max_dyn);

// Prefetch into L2 the first `count` E tiles of each of the nV vocabulary
// ranges of an LM-head launch (whole-tile split of `tiles` tiles).
// Seed scores of the starting bound of each node's top-k filter
// (csrc/dart_bound.cu): for each node n of sequence s and each of R equal
// vocabulary chunks, the score of the chunk's row of largest drafter logit
// less an error bound, ybuf[n][c]; the LM-head takes the k-th largest of a
// node's R values as its filter's starting threshold.
constexpr int kBoundMaxR = 256;
struct BoundArgs {
    int P, d, V, k, R;          // nodes per sequence, hidden, vocabulary, top-k, seed rows per sequence (multiple of 32)
    float invT;
    const float* h;             // [nseq * P][d] fp32 states
    const __nv_bfloat16* E;     // [V][d] row-major
    const float* dlog;          // drafter logits, row of sequence s: dlog + s * dlog_seq_stride + dlog_row_off
    long long dlog_seq_stride, dlog_row_off;
    float* ybuf;                // [nseq * P][R]
    int* status;
};
cudaError_t launch_seed_score(const BoundArgs& a, int nseq, cudaStream_t st);
size_t seed_score_smem(int d);
cudaError_t seed_score_set_smem_limit(int smem_optin);
int seed_score_static_smem();  // -1 on error

cudaError_t launch_lmhead_l2_prefetch(const CUtensorMap* tmE, int tiles, int nV, int d, int count, int tiled,
                                      cudaStream_t st);

// Launch plan of the tensor-core LM-head kernel for N nodes: node group NG
// (16 / 32 / 64 / 128) and G groups, nV vocabulary ranges, pipeline stages
// and dynamic shared memory; one or two CTAs per SM (ctas_per_sm_pref 1 or 2;
// 0 = two when E is streamed from its tiled copy or d <= 3072).  False if no
// plan fits the device.
struct LmheadPlan {
    int NG, G, nV, stages, smem;
};
bool plan_lmhead_tc(int N, int V, int d, int k, int num_sms, int smem_optin, int ctas_per_sm_pref, bool e_tiled,
                    LmheadPlan* out);

// fp32 CUDA-core kernels (dart_f32.cu)
cudaError_t launch_lmhead_f32(const LmheadArgs& a, cudaStream_t st);
cudaError_t launch_gemm_f32(const GemmArgs& a, cudaStream_t st);
int lmhead_f32_smem(int NG, int k);
int lmhead_f32_cw(int N);  // node columns computed for N nodes (4, 8, 16, 32)
// The whole head update (gather, W_i, SiLU, W_o, residual, RMSNorm) of Nc
// children in one launch, fp32, d <= 1024: clusters of head_small_f32_slices(d)
// blocks per child (0 = not applicable).
int head_small_f32_slices(int d);
cudaError_t launch_head_small_f32(int Nc, int d, const int* prow, const int* tok, const float* h, const float* E,
                                  const float* Wi, const float* Wo, float eps, float* hnext, cudaStream_t st);
cudaError_t f32_set_smem_limits(int max_dyn);

// selection / emission / elementwise kernels (dart_select.cu)
struct SelectArgs {
    // nV sorted key lists of klist keys per node (LM-head CTAs, or one key
    // per candidate of C_d); Pn = max |S_dep| (child slots per sequence)
    int N, P, k, nV, klist, W, L, nseq, dep, Pn;
    float beta;
    const float2* part_ms;
    const uint64_t* part_key;
    const uint64_t* gthr;  // [N] largest published k-th key per node (may be null)
    float* node_logq;      // [N][k]
    int* node_tok;         // [N][k]
    float* node_lse;       // [N]
    int* tree_tok;         // [nseq][L][W]
    int* tree_parent;
    float* tree_score;
    int* tree_count;       // [nseq][L]
    int* child_prow;       // [nseq*Pn]
    int* child_tok;
    int* seq_ticket;       // [nseq]
    int* status;
    float* lse_hist;       // optional: node n's log-sum-exp also to lse_hist[n * lse_hist_stride]
    long long lse_hist_stride;
};
cudaError_t launch_merge_select(const SelectArgs& a, cudaStream_t st);
int merge_select_smem(int nV, int klist, int k, int W);
cudaError_t select_set_smem_limits();  // the device maximum (set_max_dynamic_smem)

// candidate-restricted scoring (dart_cand.cu)
struct CandArgs {
    int K, P, d, L, dep, nseq, wbf16, V;
    float invT;
    const int* cand_tok;        // [nseq][L][K] C_d of every position, ascending tokens
    const float* dlog;          // [nseq][L][V]
    long long dlog_seq_stride;  // L * V
    long long dlog_row_off;     // (dep-1) * V
    const float* h;             // [nseq*P][d] fp32 states of S_{dep-1}
    const void* E;              // [V][d] bf16 or fp32
    float2* part_ms;            // [nseq*P][K]  (z, 1)
    uint64_t* part_key;         // [nseq*P][part_stride(K, 1)]  key(z, token)
    int DS;                     // d slices (blocks per candidate group), see cand_score_slices
    float* scratch;             // [DS][nseq*P][K] partial dot products
    int* ticket;                // [nseq][ceil(K/8)] zero between launches
};
// S = cand_topk_slices(V, K, rows, SMs) blocks per row; part: [rows][S][K]
// keys, ticket: [rows] ints, zero before the first launch (every launch
// leaves them zero).
cudaError_t launch_cand_topk(const float* dlog, int rows, int V, int K, int S, int* cand_tok, uint64_t* part,
                             int* ticket, cudaStream_t st);
// The same selection over rows of any fp32 values x [rows][V], written best
// first (value desc, index asc): tok / val [rows][out_stride], K per row.
cudaError_t launch_row_topk_by_value(const float* x, int rows, int V, int K, int S, int* tok, float* val,
                                     long long out_stride, uint64_t* part, int* ticket, cudaStream_t st);
int cand_topk_slices(int V, int K, int rows, int num_sms);
cudaError_t launch_cand_score(const CandArgs& a, cudaStream_t st);
int cand_topk_smem(int K);
int cand_score_slices(int P, int d, int nseq, int K, int max_smem);  // 0: does not fit
int cand_score_smem(int P, int d, int DS);
cudaError_t cand_set_smem_limits();    // the device maximum for both kernels

struct EmitArgs {
    int L, W, B, nseq, pos_offset;
    const int* tree_tok;
    const int* tree_parent;
    const float* tree_score;
    const int* tree_count;
    int32_t *tokens, *parents, *depths, *pos_ids, *n_nodes;
    float* scores;
    uint64_t* mask;
    int* status;
};
cudaError_t launch_prune_emit(const EmitArgs& a, cudaStream_t st);

// Best-first constructions of Table 2 (dart_heap.cu).
// Domino-chain + DDTree: the chain's best Bp children per depth (value order)
// tok / zval [nseq][L][Bp] and lse [nseq][L] -> the emitted tree.
struct DdtArgs {
    int L, B, Bp, nseq, pos_offset;
    float beta;
    const int* tok;
    const float* zval;
    const float* lse;
    int *tokens, *parents, *depths, *pos_ids, *n_nodes;
    float* scores;
    uint64_t* mask;
    int* status;
};
int ddtree_smem(int L, int Bp, int B);
cudaError_t heap_set_smem_limits();    // the device maximum
cudaError_t launch_ddtree(const DdtArgs& a, cudaStream_t st);
// Sequential correction with heap: per sequence, slot 0 = the root and slot
// p + 1 = popped node p: state tab [nseq][B+1][d], sorted children ltok / lz
// [nseq][B+1][Bp] (value order) with their log-sum-exp llse [nseq][B+1],
// cursor next and offer [nseq][B+1], pops npop [nseq]; the output rows are
// written in pop order.  hin / HL (rows s, bhalf + s): the head's input for
// the popped prefix; hout: the head's output; child_prow / child_tok /
// dlog_row [nseq]: the head update's and the LM-head's per-sequence inputs.
struct SeqHeapArgs {
    int L, B, Bp, nseq, d, pos_offset, bhalf;
    float beta;
    const float* anchor;  // [nseq][d] r_0 (slot 0 of the table)
    float* tab;
    const int* ltok;
    const float* lz;
    const float* llse;
    int* next;
    float* offer;
    int* npop;
    float* hin;
    __nv_bfloat16* HL;
    const float* hout;
    int *child_prow, *child_tok, *dlog_row;
    int *tokens, *parents, *depths, *pos_ids, *n_nodes;
    float* scores;
    uint64_t* mask;
    int* status;
};
cudaError_t launch_seqheap_step(const SeqHeapArgs& a, int t, cudaStream_t st);
cudaError_t launch_seqheap_emit(const SeqHeapArgs& a, cudaStream_t st);

// The whole round of a small fp32 problem in one cooperative kernel
// (dart_round.cu): G blocks (one per SM, at most 160), each scoring a slice
// of at most R vocabulary rows.  caps[dep] = nodes per sequence at depth dep
// (caps[0] = 1).  h0 / h1: the normalised states of odd / even depths
// [nodes][d]; rbuf, abuf [children][d]; ssqp [children][G] per-block sums of
// r^2; pms [nodes][G] and pkey [nodes][G][k] the per-slice (max, sum exp)
// and best keys; bar (kRoundBarWords words, zero: arrivals, generation and
// the one-sequence arrival ticket on separate 128-byte lines) and abort
// (zero) the grid barrier.  ecache: each block keeps its E slice in shared
// memory for the whole round; mstage: the merge stages a node's G*k keys in
// shared memory.
constexpr int kRoundMaxL = 32;
constexpr int kRoundBarWords = 96;
struct RoundArgs {
    int V, d, L, W, k, nseq, G, R;
    int ecache, mstage;
    int stage_bytes;  // cluster form: bytes of each of the two E stages (a multiple of d * 4)
    int wres;         // cluster form: each block keeps its W_i and W_o rows in shared memory
    int caps[kRoundMaxL + 1];
    float beta, invT, eps;
    const float *E, *Wi, *Wo, *dlog, *anchor;
    float *h0, *h1, *rbuf, *abuf, *ssqp;
    float2* pms;
    uint64_t* pkey;
    float *node_logq, *node_lse;
    int* node_tok;
    int *tree_tok, *tree_parent, *tree_count;
    float* tree_score;
    int *child_prow, *child_tok;
    int* status;
    unsigned* bar;
    int* abort;
    EmitArgs emit;
};
int round_small_nm(int nmax);  // node slots of the kernel instance: 4, 8, 16, 32 (0: too many)
size_t round_small_smem(int nm, int d, int R, int W, int k, int G, bool ecache, bool mstage);
cudaError_t round_small_set_smem_limits();
int round_small_blocks_per_sm(int nm, size_t smem);
cudaError_t launch_round_small_f32(const RoundArgs& a, int nm, size_t smem, cudaStream_t st);
// The same round with one cluster of kRoundCluster blocks per sequence
// (G = kRoundCluster, R = the rows of a block's vocabulary slice): pm node
// slots per sequence (4, 8, 16, 32)
constexpr int kRoundCluster = 16;
size_t round_cluster_smem(int pm, int d, int R, int W, int k, int stage_bytes, bool wres);
cudaError_t round_cluster_set_attributes();
bool round_cluster_fits(int pm, size_t smem);
size_t round_cluster_static_smem(int pm);
cudaError_t launch_round_cluster_f32(const RoundArgs& a, int pm, size_t smem, cudaStream_t st);
// two blocks at a grid barrier of three that give up after limit_ns (test hook)
cudaError_t launch_barrier_probe(unsigned* bar, int* abort, int* status, unsigned long long limit_ns,
                                 cudaStream_t st);

// bf16 [rows][cols] (row pitch `pitch` elements) -> 128 x 64 tiles, each 16 KB contiguous (tile (rt, kb)
// at index rt * cols / 64 + kb; rows past `rows` zero): every TMA request of
// the LM-head's E stream then reads one contiguous 16 KB block.
cudaError_t launch_retile(const __nv_bfloat16* src, int rows, int cols, long long pitch, __nv_bfloat16* dst,
                          cudaStream_t st);

// One CTA whose bounded mbarrier waits run out (see dart_test_wait_timeout).
cudaError_t launch_wait_probe(int* status, unsigned long long limit_ns, long long* elapsed_ns, cudaStream_t st);

// depth-1 preparation: states <- anchors, and their hi/lo bf16 split
cudaError_t launch_prep_anchor(const float* anchor, int nseq, int d, float* h, __nv_bfloat16* HL, int bhalf,
                               uint64_t* gthr_all, int n_gthr, cudaStream_t st);
// X[c] = [h[prow[c]] ; E[tok[c]]] (hi/lo bf16 or fp32)
cudaError_t launch_gather_x(int Nc, int d, const int* prow, const int* tok, const float* h, const void* E,
                            int wbf16, __nv_bfloat16* XL, int bhalf, float* X32, cudaStream_t st);
// a = SiLU(sum_s part[s]) -> AL (hi/lo) or A32
cudaError_t launch_silu_split(int Nc, int d, int S, const float* part, __nv_bfloat16* AL, int bhalf, float* A32,
                              cudaStream_t st);
// a = SiLU(Q[tok[c]] + sum_s part[s][prow[c]]) -> AL (hi/lo); part: [S][Np][d]
cudaError_t launch_gather_silu(int Nc, int d, int S, int Np, const float* part, const int* prow, const int* tok,
                               int V, const float* Q, __nv_bfloat16* AL, int bhalf, int* status, cudaStream_t st);
// debug builds (-DDART_DEBUG): one failing index check, reported through `status`
cudaError_t launch_bounds_probe(int* status, cudaStream_t st);
bool debug_build();
// h_next[c] = RMSNorm(h[prow[c]] + sum_s part[s][c]) and its hi/lo split
cudaError_t launch_residual_norm(int Nc, int d, int S, const float* part, const int* prow, const float* h,
                                 float eps, float* h_next, __nv_bfloat16* HL, int bhalf, cudaStream_t st);

}  // namespace dart
