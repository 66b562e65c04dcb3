// tcgen05 / TMA kernels of the DARTree construction path (sm_103a).
//
// One warp-specialised mainloop serves two contractions with bf16 operands
// in shared memory and fp32 accumulators in tensor memory:
//   * LM-head scoring: A = E tile [128 vocabulary rows x 64], B = node states
//     [NG nodes x 64] as hi + lo bf16 halves stored as 2*NG consecutive rows,
//     so ONE MMA with N = 2*NG computes both products (TMEM columns [0, NG)
//     = A.hi, [NG, 2NG) = A.lo; the epilogue adds them: states keep ~16
//     mantissa bits at half the MMA instruction count).  A persistent CTA
//     walks a contiguous range of vocabulary tiles; two TMEM accumulators let
//     the epilogue of tile i overlap the MMAs of tile i+1.  The epilogue adds
//     the drafter row, scales by 1/T and reduces on chip to a running
//     log-sum-exp and a top-k per node, so no [N,V] logits tensor is written.
//   * Correction-head GEMMs (split-K): A = W_i[:, 0:d] (or all of W_i) or
//     W_o tile, B = the node inputs; each CTA writes an fp32 partial tile, or
//     the k splits of a tile form a cluster that sums them on chip.  The same
//     kernel, with A = W_i[:, d:2d] and B = E rows as nodes, computes the
//     per-token table Q[t] = W_i[:, d:2d] . E[t] once per handle.
// Warp roles (192 threads): warp 0 = TMA producer, warp 1 = TMEM allocator
// and single-thread MMA issuer, warps 2-5 = epilogue (TMEM lane quarters
// warp%4).  Every wait is bounded: on timeout the CTA records kDevTimeout in
// the status word, drains its own copies/MMAs (bounded), frees TMEM and exits.
#include <algorithm>
#include <cstdio>
#include <cstdlib>

#include "dart_device.cuh"
#include "dart_kernels.h"

namespace dart {

namespace {

// 2 warps (producer, MMA) + 4 epilogue warps (one per TMEM lane quarter) per
// 16-node chunk of the group, at most 16 epilogue warps: in 128-node groups
// every epilogue warp handles two chunks.
template <int NG>
constexpr int epi_threads() {
    return 128 * (NG / 16 < 4 ? NG / 16 : 4);
}
template <int NG>
constexpr int epi_chunks() {
    return NG > 64 ? NG / 64 : 1;
}
// Candidate slots per node: a whole tile (nothing can overflow) up to 32-node
// groups; 64- and 128-node groups keep fewer (more pipeline stages fit) and
// merge in rounds when a tile overflows them.  Those groups come with the
// starting bound of the filter (seed pass before the launch), after which
// a tile rarely offers more than a few logits per node.  Measured on GB300
// at 64 nodes, k = 64 (µs per round, same box): 128 slots 3042, 64 slots
// 2806, 32 slots 2706 with the bound; without it 32 slots cost +6 %.
template <int NG>
constexpr int lm_cand_cap() {
    return NG >= 64 ? kCandCapLarge : kCandCap;
}
template <int NG>
constexpr int threads() {
    return 64 + epi_threads<NG>();
}
constexpr int kATileBytes = kTileM * kBlockK * 2;  // 16 KB

struct Work {
    int ntiles;     // consecutive A tiles handled by this CTA
    int row0;       // row coordinate of the first tile
    int kb0, kb1;   // k-block range
    int brow;       // B row of this node group (hi half); lo half at + bhalf
    int lo_kb_end;  // k-blocks >= this carry no lo half
    int tiled_kb;   // 0: A is row-major [rows][K]; else A is tiled, tile (rt, kb) at rows (rt * tiled_kb + kb) * 128
};

// TMA coordinates of A tile i (of this CTA's range), k-block kb: in the
// row-major layout (x = kb * 64, y = row), or in the tiled layout, where the
// 128 x 64 tile (rt, kb) is 16 KB of contiguous memory, viewed as rows of 64
// elements: (x = 0, y = (rt * KB + kb) * 128).
__device__ __forceinline__ int a_x(const Work& w, int kb) { return w.tiled_kb ? 0 : kb * kBlockK; }
__device__ __forceinline__ int a_y(const Work& w, int i, int kb) {
    return w.tiled_kb ? ((w.row0 / kTileM + i) * w.tiled_kb + kb) * kTileM : w.row0 + i * kTileM;
}

template <int NG>
struct Layout {
    static constexpr int kStage = kATileBytes + 2 * NG * 128;
};

__device__ __forceinline__ void record_timeout(int* status, volatile int* abort) {
    *abort = 1;
    atomicOr(status, kDevTimeout);
}

// Bounded wait that ignores the abort flag (used while draining).
__device__ __forceinline__ void drain_wait(uint64_t* bar, uint32_t parity) {
    const unsigned long long t0 = globaltimer_ns();
    while (!mbar_try_wait(bar, parity)) {
        if (globaltimer_ns() - t0 > kWaitLimitNs) return;
    }
}

template <int NG>
__device__ __forceinline__ void producer(const CUtensorMap* tmA, const CUtensorMap* tmB, const Work& w, int bhalf,
                                         uint8_t* ring, int stages, uint64_t* full, uint64_t* empty,
                                         volatile int* abort, int* status, int l2pf = 0, bool keep_a = false) {
    // A: streamed once (E), or kept for the next depth (head weights when
    // nothing else streams through L2)
    const uint64_t pol_a = keep_a ? l2_policy_evict_last() : l2_policy_evict_first();
    const uint64_t pol_b = l2_policy_evict_last();   // re-read by every tile
    const int kbs = w.kb1 - w.kb0;
    const uint32_t total = static_cast<uint32_t>(w.ntiles * kbs);
    // The A operand (E or a head weight) never depends on an earlier kernel:
    // its first `pre` stages are requested before waiting on the previous
    // kernel; the B operand (node states) only after.
    const uint32_t pre = total < static_cast<uint32_t>(stages) ? total : static_cast<uint32_t>(stages);
    for (uint32_t f = 0; f < pre; f++) {
        const int i = static_cast<int>(f) / kbs, kb = w.kb0 + static_cast<int>(f) % kbs;
        const bool lo = kb < w.lo_kb_end;
        mbar_arrive_expect_tx(&full[f], kATileBytes + NG * 128 * (lo ? 2 : 1));
        tma_load_2d(ring + f * Layout<NG>::kStage, tmA, &full[f], a_x(w, kb), a_y(w, i, kb), pol_a);
    }
    // and the next `l2pf` into L2, while the previous kernel still runs
    for (uint32_t f = pre; f < pre + static_cast<uint32_t>(l2pf) && f < total; f++) {
        const int i = static_cast<int>(f) / kbs, kb = w.kb0 + static_cast<int>(f) % kbs;
        tma_prefetch_2d(tmA, a_x(w, kb), a_y(w, i, kb));
    }
    pdl_wait();
    for (uint32_t f = 0; f < pre; f++) {
        const int kb = w.kb0 + static_cast<int>(f) % kbs;
        uint8_t* sH = ring + f * Layout<NG>::kStage + kATileBytes;
        tma_load_2d(sH, tmB, &full[f], kb * kBlockK, w.brow, pol_b);
        if (kb < w.lo_kb_end) tma_load_2d(sH + NG * 128, tmB, &full[f], kb * kBlockK, bhalf + w.brow, pol_b);
    }
    uint32_t stage = pre % stages, phase = (pre / stages) & 1u, fills = pre;
    bool ok = true;
    for (uint32_t f = pre; f < total; f++) {
        if (!mbar_wait(&empty[stage], phase ^ 1u, abort)) {
            record_timeout(status, abort);
            ok = false;
            break;
        }
        const int i = static_cast<int>(f) / kbs, kb = w.kb0 + static_cast<int>(f) % kbs;
        const bool lo = kb < w.lo_kb_end;
        uint8_t* sA = ring + stage * Layout<NG>::kStage;
        uint8_t* sH = sA + kATileBytes;
        mbar_arrive_expect_tx(&full[stage], kATileBytes + NG * 128 * (lo ? 2 : 1));
        tma_load_2d(sA, tmA, &full[stage], a_x(w, kb), a_y(w, i, kb), pol_a);
        tma_load_2d(sH, tmB, &full[stage], kb * kBlockK, w.brow, pol_b);
        if (lo) tma_load_2d(sH + NG * 128, tmB, &full[stage], kb * kBlockK, bhalf + w.brow, pol_b);
        fills++;
        if (++stage == static_cast<uint32_t>(stages)) {
            stage = 0;
            phase ^= 1u;
        }
    }
    if (!ok) {
        // wait for this thread's copies still in flight before the CTA exits
        const uint32_t first = fills > static_cast<uint32_t>(stages) ? fills - stages : 0;
        for (uint32_t f = first; f < fills; f++) drain_wait(&full[f % stages], (f / stages) & 1u);
    }
}

template <int NG>
__device__ __forceinline__ void mma_issuer(const Work& w, uint8_t* ring, int stages, uint64_t* full,
                                           uint64_t* empty, uint64_t* tfull, uint64_t* tempty, uint64_t* tdown,
                                           uint32_t tmem_base, int acc_stride, volatile int* abort,
                                           int* status, int nacc = 2) {
    constexpr uint32_t idesc2 = idesc_bf16_f32(kTileM, 2 * NG);  // hi and lo rows together
    constexpr uint32_t idesc1 = idesc_bf16_f32(kTileM, NG);      // hi rows only (no lo half)
    uint32_t stage = 0, phase = 0;
    bool ok = true;
    for (int i = 0; i < w.ntiles && ok; i++) {
        const int acc = i % nacc;
        const uint32_t aph = (i / nacc) & 1;
        if (!mbar_wait(&tempty[acc], aph ^ 1u, abort)) {
            record_timeout(status, abort);
            ok = false;
            break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * acc_stride;
        for (int kb = w.kb0; kb < w.kb1; kb++) {
            if (!mbar_wait(&full[stage], phase, abort)) {
                record_timeout(status, abort);
                ok = false;
                break;
            }
            tc_fence_after();
            const uint32_t idesc = kb < w.lo_kb_end ? idesc2 : idesc1;
            const uint32_t a = smem_u32(ring + stage * Layout<NG>::kStage);
            const uint32_t hb = a + kATileBytes;
#pragma unroll
            for (int kk = 0; kk < kBlockK / 16; kk++)
                tc_mma_bf16(d_tmem, sdesc_sw128(a + kk * 32), sdesc_sw128(hb + kk * 32), idesc,
                            (kb > w.kb0 || kk > 0) ? 1u : 0u);
            tc_commit(&empty[stage]);  // frees the smem stage once these MMAs are done
            if (++stage == static_cast<uint32_t>(stages)) {
                stage = 0;
                phase ^= 1u;
            }
        }
        if (ok) tc_commit(&tfull[acc]);
    }
    if (!ok) {
        // make sure no MMA still reads smem / writes TMEM before teardown
        tc_commit(tdown);
        drain_wait(tdown, 0);
    }
}

struct Smem {
    uint8_t* ring;
    uint64_t *full, *empty, *tfull, *tempty, *tdown;
    int* misc;  // [0] tmem base, [1] abort flag, [2] epilogue flag
    uint8_t* tail;
};

template <int NG>
__device__ __forceinline__ Smem carve(uint8_t* raw, int stages, int nacc = 2) {
    Smem s;
    const uint32_t off = (1024u - (smem_u32(raw) & 1023u)) & 1023u;
    s.ring = raw + off;
    s.full = reinterpret_cast<uint64_t*>(s.ring + stages * Layout<NG>::kStage);
    s.empty = s.full + stages;
    s.tfull = s.empty + stages;
    s.tempty = s.tfull + nacc;
    s.tdown = s.tempty + nacc;
    s.misc = reinterpret_cast<int*>(s.tdown + 1);
    s.tail = reinterpret_cast<uint8_t*>(s.misc + 4);
    return s;
}

template <int NG>
__device__ __forceinline__ uint32_t setup(const Smem& s, int stages, int ncols, int nacc = 2) {
    constexpr int kEpi = epi_threads<NG>();
    const int warp = threadIdx.x >> 5;
    if (threadIdx.x == 0) {
        for (int i = 0; i < stages; i++) {
            mbar_init(&s.full[i], 1);
            mbar_init(&s.empty[i], 1);
        }
        for (int i = 0; i < nacc; i++) {
            mbar_init(&s.tfull[i], 1);
            mbar_init(&s.tempty[i], kEpi);
        }
        mbar_init(s.tdown, 1);
        s.misc[1] = 0;
        s.misc[2] = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(reinterpret_cast<uint32_t*>(&s.misc[0]), ncols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    return static_cast<uint32_t>(s.misc[0]);
}

__device__ __forceinline__ void teardown(uint32_t tmem_base, int ncols) {
    tc_fence_before();
    __syncthreads();
    if ((threadIdx.x >> 5) == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem_base, ncols);
    }
}

// One accumulator = 2*NG fp32 columns (hi products, then lo products).
template <int NG>
constexpr int acc_stride() {
    return 2 * NG < 32 ? 32 : 2 * NG;
}
template <int NG>
constexpr int tmem_cols() {
    return 2 * acc_stride<NG>() <= 32 ? 32
                                      : (2 * acc_stride<NG>() <= 64 ? 64
                                                                    : (2 * acc_stride<NG>() <= 128
                                                                           ? 128
                                                                           : (2 * acc_stride<NG>() <= 256 ? 256 : 512)));
}

// Accumulators of the LM-head (a ring in TMEM): with 64-node groups four,
// so that the MMAs run up to three tiles ahead of the epilogue, whose cost
// per tile is uneven (the first tiles of a vocabulary range pass most
// logits to the top-k merges, later ones few).  All of TMEM then belongs to
// one CTA, which the plan's shared memory makes the only LM-head CTA of its SM.
template <int NG>
constexpr int lm_nacc() {
    return NG == 64 ? 4 : 2;
}
template <int NG>
constexpr int lm_tmem_cols() {
    return lm_nacc<NG>() * acc_stride<NG>() <= 32
               ? 32
               : (lm_nacc<NG>() * acc_stride<NG>() <= 64
                      ? 64
                      : (lm_nacc<NG>() * acc_stride<NG>() <= 128 ? 128
                                                                 : (lm_nacc<NG>() * acc_stride<NG>() <= 256 ? 256 : 512)));
}

// ------------------------------------------------------------ LM-head kernel

template <int NG>
__global__ void __launch_bounds__(threads<NG>(), 1)
    lmhead_tc_kernel(const __grid_constant__ CUtensorMap tmE, const __grid_constant__ CUtensorMap tmH,
                     const LmheadArgs a) {
    extern __shared__ uint8_t smem_raw[];
    pdl_trigger();
    const int stages = a.stages;
    constexpr int kNacc = lm_nacc<NG>();
    Smem s = carve<NG>(smem_raw, stages, kNacc);
    constexpr int kCap = lm_cand_cap<NG>();
    EpiSmem e;
    e.cap = kCap;
    e.list = reinterpret_cast<uint64_t*>(s.tail);
    e.cand = e.list + NG * a.k;
    e.gcache = e.cand + NG * kCap;
    e.stats = reinterpret_cast<float2*>(e.gcache + NG);
    e.mref = reinterpret_cast<float*>(e.stats + 4 * NG);
    e.cnt = reinterpret_cast<int*>(e.mref + 4 * NG);
    e.more = e.cnt + NG;

    const int g = blockIdx.x % a.G;
    const int vr = blockIdx.x / a.G;
    const int t0 = static_cast<int>((static_cast<long long>(vr) * a.tiles) / a.nV);
    const int t1 = static_cast<int>((static_cast<long long>(vr + 1) * a.tiles) / a.nV);
    Work w;
    w.ntiles = t1 - t0;
    w.row0 = t0 * kTileM;
    w.kb0 = 0;
    w.kb1 = a.d / kBlockK;
    w.brow = g * NG;
    w.lo_kb_end = w.kb1;
    w.tiled_kb = a.e_tiled ? w.kb1 : 0;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t tmem_base = setup<NG>(s, stages, lm_tmem_cols<NG>(), kNacc);
    volatile int* abort = &s.misc[1];

    if (warp == 0) {
        if (lane == 0)
            producer<NG>(&tmE, &tmH, w, a.bhalf, s.ring, stages, s.full, s.empty, abort, a.status, a.l2pf);
    } else if (warp == 1) {
        if (lane == 0)
            mma_issuer<NG>(w, s.ring, stages, s.full, s.empty, s.tfull, s.tempty, s.tdown, tmem_base,
                           acc_stride<NG>(), abort, a.status, kNacc);
    } else {
        // epilogue warp wi = warp - 2 reads TMEM lane quarter warp % 4 and
        // owns the 16-node chunks wi / 4 + 4 * ci (ci < kChunks) of the group
        constexpr int kEpi = epi_threads<NG>();
        constexpr int kChunks = epi_chunks<NG>();
        const int etid = threadIdx.x - 64;
        const int wi = warp - 2;
        const int quarter = warp & 3;
        pdl_wait();
        epi_init(e, NG, a.k, etid, kEpi, a.gthr, g * NG, a.N, a.seed_y, a.seed_R, vr == 0);
        float ssum[kChunks];
        uint32_t nodemask[kChunks];
#pragma unroll
        for (int ci = 0; ci < kChunks; ci++) {
            const int c0 = ((wi >> 2) + 4 * ci) * 16;
            ssum[ci] = 0.0f;
            nodemask[ci] = 0;
            for (int j = 0; j < 16; j++)
                if (g * NG + c0 + j < a.N) nodemask[ci] |= 1u << j;
        }
        // scaled logits of this thread's row v for chunk ci from accumulator acc:
        // hi + lo products, drafter row added, 1/T applied
        auto load_z = [&](int acc, int ci, int v, bool valid, float (&z)[16]) {
            const int c0 = ((wi >> 2) + 4 * ci) * 16;
            float zl[16];
            const uint32_t tcol =
                tmem_base + acc * acc_stride<NG>() + c0 + (static_cast<uint32_t>(quarter * 32) << 16);
            tmem_ld16_pair(tcol, tcol + NG, z, zl);
#pragma unroll
            for (int j = 0; j < 16; j++) z[j] += zl[j];
            int cur_seq = -1;
            float dl = 0.0f;
#pragma unroll
            for (int j = 0; j < 16; j++) {
                if ((nodemask[ci] >> j) & 1u) {
                    const int seq = (g * NG + c0 + j) / a.P;
                    if (seq != cur_seq) {
                        cur_seq = seq;
                        const long long off = a.dlog_row ? static_cast<long long>(__ldg(a.dlog_row + seq)) * a.V
                                                         : a.dlog_row_off;
                        dl = valid ? __ldg(a.dlog + seq * a.dlog_seq_stride + off + v) : 0.0f;
                    }
                    z[j] = (z[j] + dl) * a.invT;
                }
            }
        };
        for (int i = 0; i < w.ntiles; i++) {
            const int acc = i % kNacc;
            const uint32_t aph = (i / kNacc) & 1;
            if (etid == 0) {
                const bool ok = mbar_wait(&s.tfull[acc], aph, abort);
                if (!ok) record_timeout(a.status, abort);
                s.misc[2] = ok ? 1 : 0;
            }
            named_bar_sync(kEpiBarrier, kEpi);
            if (s.misc[2] == 0) break;
            tc_fence_after();
            const int v = w.row0 + i * kTileM + quarter * 32 + lane;
            const bool valid = v < a.V;
            if constexpr (kCap >= kTileM) {
                // every candidate of the tile fits: one merge, and the
                // accumulator is released as soon as it has been read
                float z[16];
                load_z(acc, 0, v, valid, z);
                tc_fence_before();
                mbar_arrive(&s.tempty[acc]);
                if (a.zout && valid) {
                    const int nb = g * NG + (wi >> 2) * 16;
#pragma unroll
                    for (int j = 0; j < 16; j++)
                        if ((nodemask[0] >> j) & 1u) a.zout[static_cast<long long>(nb + j) * a.zout_stride + v] = z[j];
                }
                (void)epi_chunk(e, NG, a.k, quarter, lane, (wi >> 2) * 16, z, nodemask[0], valid,
                                static_cast<uint32_t>(v), ssum[0]);
                epi_merge(e, NG, a.k, wi, lane, kEpi, etid, a.gthr, g * NG, a.N);
            } else {
                uint32_t pend[kChunks];
#pragma unroll
                for (int ci = 0; ci < kChunks; ci++) {
                    float z[16];
                    load_z(acc, ci, v, valid, z);
                    pend[ci] = epi_chunk(e, NG, a.k, quarter, lane, ((wi >> 2) + 4 * ci) * 16, z, nodemask[ci],
                                         valid, static_cast<uint32_t>(v), ssum[ci]);
                }
                // Merge rounds while some candidate found no free slot: those
                // still beating the raised thresholds are read again from the
                // accumulator (kept until the last round) and offered again.
                // A round's flag is set before epi_merge's first barrier, read
                // after its second, and cleared in the next round after that
                // round's first barrier.
                for (int round = 0;; round++) {
                    bool any = false;
#pragma unroll
                    for (int ci = 0; ci < kChunks; ci++) any |= pend[ci] != 0u;
                    if (__any_sync(kFull, any) && lane == 0) atomicOr(&e.more[round & 1], 1);
                    epi_merge(e, NG, a.k, wi, lane, kEpi, etid, a.gthr, g * NG, a.N,
                              round > 0 ? &e.more[(round + 1) & 1] : nullptr);
                    if (e.more[round & 1] == 0) break;
#pragma unroll
                    for (int ci = 0; ci < kChunks; ci++) {
                        if (__any_sync(kFull, pend[ci] != 0u)) {
                            const int c0 = ((wi >> 2) + 4 * ci) * 16;
                            float z[16];
                            load_z(acc, ci, v, valid, z);
                            pend[ci] = epi_offer(e, c0, z, epi_still_pass(e, a.k, c0, z, pend[ci], static_cast<uint32_t>(v)),
                                                 static_cast<uint32_t>(v), lane);
                        }
                    }
                }
                tc_fence_before();
                mbar_arrive(&s.tempty[acc]);
            }
        }
#pragma unroll
        for (int ci = 0; ci < kChunks; ci++) epi_stash(e, NG, quarter, lane, ((wi >> 2) + 4 * ci) * 16, ssum[ci]);
        epi_finalize(e, NG, a.k, etid, kEpi, g * NG, a.N, vr, a.nV, a.part_ms, a.part_key);
    }
    teardown(tmem_base, lm_tmem_cols<NG>());
}

// --------------------------------------------------------------- GEMM kernel
//
// Correction-head layer out = A . B^T with A = W_i or W_o [M x K] and B the
// node inputs [N x K], split over K into a.S parts.
//   kGemmPartials:  every CTA writes its fp32 partial tile to out[split]; the
//                   elementwise kernels that follow sum the splits.
//   kGemmSiluSplit, kGemmSum: the S splits of one (M tile, node group) form
//                   a thread-block cluster: every CTA stages its fp32 tile in
//                   shared memory, and after a cluster barrier CTA r sums
//                   rows [r*R, (r+1)*R) of the tile over the S CTAs in rank
//                   order (deterministic) and writes outL = hi/lo bf16 split
//                   of SiLU(sum) (input of W_o), or out = sum in fp32.

template <int NG>
__global__ void __launch_bounds__(threads<NG>(), 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const GemmArgs a) {
    extern __shared__ uint8_t smem_raw[];
    pdl_trigger();
    const int stages = a.stages;
    Smem s = carve<NG>(smem_raw, stages);

    // block = (g * MT + mt) * S + split: the S splits of a tile are consecutive,
    // i.e. one cluster
    const int tile = blockIdx.x / a.S;
    const int mt_c = tile % a.MT, g_c = tile / a.MT, split_c = blockIdx.x % a.S;
    Work w;
    w.ntiles = 1;
    w.row0 = mt_c * kTileM;
    w.kb0 = static_cast<int>((static_cast<long long>(split_c) * a.KB) / a.S);
    w.kb1 = static_cast<int>((static_cast<long long>(split_c + 1) * a.KB) / a.S);
    w.brow = g_c * NG;
    w.lo_kb_end = a.lo_kb_end;
    w.tiled_kb = a.a_tiled_kb;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t tmem_base = setup<NG>(s, stages, tmem_cols<NG>());
    volatile int* abort = &s.misc[1];
    // staging tile [NG nodes][128 rows] fp32, in the pipeline ring (free once
    // the last MMA has completed)
    float* stage_tile = reinterpret_cast<float*>(s.ring);

    if (warp == 0) {
        if (lane == 0)
            producer<NG>(&tmA, &tmB, w, a.bhalf, s.ring, stages, s.full, s.empty, abort, a.status, 0, a.keep_a != 0);
    } else if (warp == 1) {
        if (lane == 0)
            mma_issuer<NG>(w, s.ring, stages, s.full, s.empty, s.tfull, s.tempty, s.tdown, tmem_base,
                           acc_stride<NG>(), abort, a.status);
    } else {
        const int etid = threadIdx.x - 64;
        const int quarter = warp & 3;
        pdl_wait();
        if (etid == 0) {
            const bool ok = mbar_wait(&s.tfull[0], 0, abort);
            if (!ok) record_timeout(a.status, abort);
            s.misc[2] = ok ? 1 : 0;
        }
        named_bar_sync(kEpiBarrier, epi_threads<NG>());
        if (s.misc[2] != 0) {
            tc_fence_after();
            const int c0 = ((warp - 2) >> 2) * 16;
            float vals[16], lov[16];
            const uint32_t tcol = tmem_base + c0 + (static_cast<uint32_t>(quarter * 32) << 16);
            tmem_ld16_pair(tcol, tcol + NG, vals, lov);
            // lo columns were written only if this split saw a k-block with a lo half
            if (w.kb0 < w.lo_kb_end) {
#pragma unroll
                for (int j = 0; j < 16; j++) vals[j] += lov[j];
            }
            if (a.mode == kGemmPartials) {
                const int m = w.row0 + quarter * 32 + lane;
                float* out = a.out + static_cast<size_t>(split_c) * a.N * a.M;
#pragma unroll
                for (int j = 0; j < 16; j++) {
                    const int n = g_c * NG + c0 + j;
                    if (m < a.M && n < a.N) out[static_cast<size_t>(n) * a.M + m] = vals[j];
                }
            } else {
#pragma unroll
                for (int j = 0; j < 16; j++) stage_tile[(c0 + j) * kTileM + quarter * 32 + lane] = vals[j];
            }
        }
    }
    teardown(tmem_base, tmem_cols<NG>());
    if (a.mode == kGemmPartials) return;  // launched without clusters
    cluster_sync_all();  // every split's tile is staged
    {
        const int S = a.S;
        const uint32_t r = cluster_ctarank();
        const int R = (kTileM + S - 1) / S;
        const int nthr = threads<NG>();
        const uint32_t base = smem_u32(stage_tile);
        for (int idx = threadIdx.x; idx < R * NG; idx += nthr) {
            const int nl = idx / R, row = static_cast<int>(r) * R + idx % R;
            const int m = w.row0 + row, n = g_c * NG + nl;
            if (row >= kTileM || m >= a.M || n >= a.N) continue;
            const uint32_t off = base + static_cast<uint32_t>((nl * kTileM + row) * 4);
            float v[kMaxClusterK];
#pragma unroll
            for (int q = 0; q < kMaxClusterK; q++) v[q] = q < S ? ld_cluster_f32(off, static_cast<uint32_t>(q)) : 0.0f;
            float acc = 0.0f;
#pragma unroll
            for (int q = 0; q < kMaxClusterK; q++)
                if (q < S) acc += v[q];
            const size_t o = static_cast<size_t>(n) * a.M + m;
            if (a.mode == kGemmSiluSplit) {
                const float act = acc / (1.0f + expf(-acc));
                __nv_bfloat16 hi, lo;
                split_bf16(act, hi, lo);
                a.outL[o] = hi;
                a.outL[static_cast<size_t>(a.bhalf) * a.M + o] = lo;
            } else {
                a.out[o] = acc;
            }
        }
    }
    cluster_sync_all();  // no CTA leaves while a peer still reads its staging tile
}

template <int NG>
int lmhead_fixed(int k, int stages) {
    return (2 * stages + 2 * lm_nacc<NG>() + 1) * 8 + 16 + NG * k * 8 + NG * lm_cand_cap<NG>() * 8 + NG * 8 + 4 * NG * 8 + 4 * NG * 4 +
           NG * 4 + 8;
}

// The failure path of the bounded waits, exercised without a fault: two
// mbarriers that nothing ever completes (count 1, no arrival, no copy or MMA
// tracked by them).  Thread 0 waits with limit_ns, gives up and records the
// timeout exactly as the pipeline roles do (abort flag + status bit); thread
// 32 waits with the kernels' own limit and returns once it sees the abort
// flag.  Each records how long its wait took.
__global__ void __launch_bounds__(64) wait_probe_kernel(int* status, unsigned long long limit_ns,
                                                        long long* elapsed_ns) {
    __shared__ __align__(8) uint64_t bar[2];
    __shared__ int abort_flag;
    if (threadIdx.x == 0) {
        mbar_init(&bar[0], 1);
        mbar_init(&bar[1], 1);
        abort_flag = 0;
        fence_mbar_init();
    }
    __syncthreads();
    volatile int* abort = &abort_flag;
    const unsigned long long t0 = globaltimer_ns();
    long long took = -1;
    if (threadIdx.x == 0) {
        if (!mbar_wait(&bar[0], 0, abort, limit_ns)) record_timeout(status, abort);
        took = static_cast<long long>(globaltimer_ns() - t0);
    } else if (threadIdx.x == 32) {
        if (!mbar_wait(&bar[1], 0, abort)) took = static_cast<long long>(globaltimer_ns() - t0);
    }
    if (elapsed_ns && took >= 0) elapsed_ns[threadIdx.x == 0 ? 0 : 1] = took;
}

template <int NG>
cudaError_t launch_lmhead_ng(const CUtensorMap* tmE, const CUtensorMap* tmH, const LmheadArgs& a, int smem,
                             cudaStream_t st) {
    return launch_pdl(lmhead_tc_kernel<NG>, dim3(a.nV * a.G), dim3(threads<NG>()), smem, st, *tmE, *tmH, a);
}
template <int NG>
cudaError_t launch_gemm_ng(const CUtensorMap* tmA, const CUtensorMap* tmB, const GemmArgs& a, int smem,
                           cudaStream_t st) {
    if (a.mode == kGemmPartials)
        return launch_pdl(gemm_tc_kernel<NG>, dim3(a.MT * a.G * a.S), dim3(threads<NG>()), smem, st, *tmA, *tmB, a);
    return launch_pdl_cluster(gemm_tc_kernel<NG>, dim3(a.MT * a.G * a.S), dim3(threads<NG>()), smem, st, a.S, *tmA,
                              *tmB, a);
}

template <int NG>
int max_clusters_ng(int smem, int cluster) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(cluster * 1024);
    cfg.blockDim = dim3(threads<NG>());
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = static_cast<unsigned>(cluster);
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, gemm_tc_kernel<NG>, &cfg) != cudaSuccess) {
        cudaGetLastError();
        return 0;
    }
    return n;
}

}  // namespace

int tc_stage_bytes(int NG) { return kATileBytes + 2 * NG * 128; }

int lmhead_tc_tmem_cols(int NG) {
    switch (NG) {
        case 16: return lm_tmem_cols<16>();
        case 32: return lm_tmem_cols<32>();
        case 64: return lm_tmem_cols<64>();
        default: return lm_tmem_cols<128>();
    }
}

int lmhead_tc_fixed_smem(int NG, int k, int stages) {
    switch (NG) {
        case 16: return lmhead_fixed<16>(k, stages) + 1024;
        case 32: return lmhead_fixed<32>(k, stages) + 1024;
        case 64: return lmhead_fixed<64>(k, stages) + 1024;
        default: return lmhead_fixed<128>(k, stages) + 1024;
    }
}

int gemm_tc_fixed_smem(int stages) { return (2 * stages + 5) * 8 + 16 + 1024; }

// Resident CTAs per SM for a kernel with `smem` bytes of dynamic shared
// memory, from the device limits (shared memory with the per-block
// reservation, register file at 8-register granularity, threads).
static int ctas_per_sm(const void* fn, int nthreads, int smem) {
    int dev = 0, sm_smem = 0, reserved = 0, sm_regs = 0, sm_threads = 0;
    cudaFuncAttributes fa;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaFuncGetAttributes(&fa, fn) != cudaSuccess ||
        cudaDeviceGetAttribute(&sm_smem, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&reserved, cudaDevAttrReservedSharedMemoryPerBlock, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sm_regs, cudaDevAttrMaxRegistersPerMultiprocessor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sm_threads, cudaDevAttrMaxThreadsPerMultiProcessor, dev) != cudaSuccess)
        return 1;
    const int per_smem = smem + static_cast<int>(fa.sharedSizeBytes) + reserved;
    const int per_regs = ((fa.numRegs + 7) / 8) * 8 * nthreads;
    int n = per_smem > 0 ? sm_smem / per_smem : 1;
    if (per_regs > 0) n = std::min(n, sm_regs / per_regs);
    n = std::min(n, sm_threads / nthreads);
    return std::max(n, 1);
}

int gemm_tc_ctas_per_sm(int NG, int smem) {
    switch (NG) {
        case 16: return ctas_per_sm(reinterpret_cast<const void*>(gemm_tc_kernel<16>), threads<16>(), smem);
        case 32: return ctas_per_sm(reinterpret_cast<const void*>(gemm_tc_kernel<32>), threads<32>(), smem);
        default: return ctas_per_sm(reinterpret_cast<const void*>(gemm_tc_kernel<64>), threads<64>(), smem);
    }
}

int gemm_tc_max_clusters(int NG, int smem, int cluster) {
    switch (NG) {
        case 16: return max_clusters_ng<16>(smem, cluster);
        case 32: return max_clusters_ng<32>(smem, cluster);
        default: return max_clusters_ng<64>(smem, cluster);
    }
}

int lmhead_tc_ctas_per_sm(int NG, int smem) {
    switch (NG) {
        case 16: return ctas_per_sm(reinterpret_cast<const void*>(lmhead_tc_kernel<16>), threads<16>(), smem);
        case 32: return ctas_per_sm(reinterpret_cast<const void*>(lmhead_tc_kernel<32>), threads<32>(), smem);
        case 64: return ctas_per_sm(reinterpret_cast<const void*>(lmhead_tc_kernel<64>), threads<64>(), smem);
        default: return ctas_per_sm(reinterpret_cast<const void*>(lmhead_tc_kernel<128>), threads<128>(), smem);
    }
}

bool plan_lmhead_tc(int N, int V, int d, int k, int num_sms, int smem_optin, int ctas_per_sm_pref, bool e_tiled,
                    LmheadPlan* out) {
    LmheadPlan p;
    p.NG = N <= 16 ? 16 : (N <= 32 ? 32 : (N <= 64 ? 64 : 128));
    p.G = (N + p.NG - 1) / p.NG;
    const int tiles = (V + kTileM - 1) / kTileM;
    p.nV = std::max(1, std::min(num_sms / p.G, tiles));
    const int sb = tc_stage_bytes(p.NG);
    const int fixed = lmhead_tc_fixed_smem(p.NG, k, 16);
    auto stages_in = [&](int budget) { return std::min(16, (budget - fixed) / sb); };
    // Two CTAs per SM when both fit with >= 4 pipeline stages each: two
    // independent TMA streams per SM, and one CTA's epilogue / start-up /
    // tail overlaps the other's stream.  Measured on GB300 (A/B per round):
    // with E row-major it pays for short rows (d = 2560: -4 %) but not for
    // d = 4096 (+6 %), where the deeper single-CTA pipeline wins; with E in
    // contiguous 16 KB tiles two CTAs win at d = 4096 too (-3.6 % against
    // one CTA on the same tiles, -1.0 % against row-major with one).
    const int st2 = stages_in(smem_optin / 2 - 2048);
    const int smem2 = lmhead_tc_fixed_smem(p.NG, k, st2) + st2 * sb;
    const bool want2 = ctas_per_sm_pref ? ctas_per_sm_pref == 2 : (e_tiled || d <= 3072);
    if (want2 && st2 >= 4 && 2 * lmhead_tc_tmem_cols(p.NG) <= 512 && lmhead_tc_ctas_per_sm(p.NG, smem2) >= 2) {
        p.stages = st2;
        p.nV = std::max(1, std::min(2 * num_sms / p.G, tiles));
    } else {
        p.stages = stages_in(smem_optin);
    }
    if (p.stages < 2) return false;
    p.smem = lmhead_tc_fixed_smem(p.NG, k, p.stages) + p.stages * sb;
    *out = p;
    return true;
}

cudaError_t tc_set_smem_limits(int max_dyn) {
    cudaError_t e = cudaSuccess;
#define DART_SET(fn)                                                                                   \
    if (e == cudaSuccess) e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, max_dyn); \
    if (e == cudaSuccess)                                                                              \
        e = cudaFuncSetAttribute(fn, cudaFuncAttributePreferredSharedMemoryCarveout, cudaSharedmemCarveoutMaxShared);
    DART_SET(lmhead_tc_kernel<16>)
    DART_SET(lmhead_tc_kernel<32>)
    DART_SET(lmhead_tc_kernel<64>)
    DART_SET(lmhead_tc_kernel<128>)
    DART_SET(gemm_tc_kernel<16>)
    DART_SET(gemm_tc_kernel<32>)
    DART_SET(gemm_tc_kernel<64>)
#undef DART_SET
    return e;
}

cudaError_t launch_lmhead_tc(const CUtensorMap* tmE, const CUtensorMap* tmH, const LmheadArgs& a, int smem,
                             cudaStream_t st) {
    switch (a.NG) {
        case 16: return launch_lmhead_ng<16>(tmE, tmH, a, smem, st);
        case 32: return launch_lmhead_ng<32>(tmE, tmH, a, smem, st);
        case 64: return launch_lmhead_ng<64>(tmE, tmH, a, smem, st);
        case 128: return launch_lmhead_ng<128>(tmE, tmH, a, smem, st);
        default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_gemm_tc(const CUtensorMap* tmA, const CUtensorMap* tmB, const GemmArgs& a, int smem,
                           cudaStream_t st) {
    switch (a.NG) {
        case 16: return launch_gemm_ng<16>(tmA, tmB, a, smem, st);
        case 32: return launch_gemm_ng<32>(tmA, tmB, a, smem, st);
        case 64: return launch_gemm_ng<64>(tmA, tmB, a, smem, st);
        default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_wait_probe(int* status, unsigned long long limit_ns, long long* elapsed_ns, cudaStream_t st) {
    wait_probe_kernel<<<1, 64, 0, st>>>(status, limit_ns, elapsed_ns);
    return cudaGetLastError();
}

namespace {

// dst = src [rows][cols] bf16 (row pitch `pitch`) re-laid as 128 x 64 tiles, tile (rt, kb)
// (rows 128 rt .., columns 64 kb ..) as 16 KB of contiguous memory at tile
// index rt * (cols / 64) + kb, rows 128-byte, rows past `rows` zero.  One
// thread per 16-byte chunk of dst.
__global__ void retile_kernel(const __nv_bfloat16* src, int rows, int cols, long long pitch, __nv_bfloat16* dst,
                              long long chunks) {
    const int KB = cols / kBlockK;
    for (long long q = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; q < chunks;
         q += static_cast<long long>(gridDim.x) * blockDim.x) {
        const int c8 = static_cast<int>(q & 7);
        const int r = static_cast<int>((q >> 3) & (kTileM - 1));
        const long long tile = q >> 10;
        const long long rt = tile / KB;
        const int kb = static_cast<int>(tile % KB);
        const long long row = rt * kTileM + r;
        uint4 v = make_uint4(0u, 0u, 0u, 0u);
        if (row < rows) v = *reinterpret_cast<const uint4*>(src + row * pitch + kb * kBlockK + c8 * 8);
        reinterpret_cast<uint4*>(dst)[q] = v;
    }
}

}  // namespace

cudaError_t launch_retile(const __nv_bfloat16* src, int rows, int cols, long long pitch, __nv_bfloat16* dst,
                          cudaStream_t st) {
    const long long rt = (rows + kTileM - 1) / kTileM;
    const long long chunks = rt * (cols / kBlockK) * kTileM * 8;
    retile_kernel<<<4096, 256, 0, st>>>(src, rows, cols, pitch, dst, chunks);
    return cudaGetLastError();
}

namespace {

// The first `count` E tiles of every CTA of an LM-head launch (nV vocabulary
// ranges of whole tiles, the same split as lmhead_tc_kernel) prefetched into
// L2, one block per range so that every SM's TMA unit issues its own share
// (one unit issuing them all takes hundreds of microseconds).  Launched beside
// the selection of the previous depth, while HBM would otherwise wait.
__global__ void lmhead_l2_prefetch_kernel(const __grid_constant__ CUtensorMap tmE, int tiles, int nV, int KB, int count,
                                          int tiled) {
    const int vr = blockIdx.x;
    if (threadIdx.x != 0 || vr >= nV) return;
    const int t0 = static_cast<int>((static_cast<long long>(vr) * tiles) / nV);
    const int t1 = static_cast<int>((static_cast<long long>(vr + 1) * tiles) / nV);
    Work w;
    w.ntiles = t1 - t0;
    w.row0 = t0 * kTileM;
    w.kb0 = 0;
    w.kb1 = KB;
    w.brow = 0;
    w.lo_kb_end = KB;
    w.tiled_kb = tiled ? KB : 0;
    const int total = w.ntiles * KB;
    for (int f = 0; f < count && f < total; f++) tma_prefetch_2d(&tmE, a_x(w, f % KB), a_y(w, f / KB, f % KB));
}

}  // namespace

cudaError_t launch_lmhead_l2_prefetch(const CUtensorMap* tmE, int tiles, int nV, int d, int count, int tiled,
                                      cudaStream_t st) {
    const int KB = d / kBlockK;
    lmhead_l2_prefetch_kernel<<<nV, 32, 0, st>>>(*tmE, tiles, nV, KB, count, tiled);
    return cudaGetLastError();
}

}  // namespace dart
