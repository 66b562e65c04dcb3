// Tree-attention verification consumer of the emitted draft tree (Sec. 2.2,
// "Tree Verification and DDTree": every flattened tree node attends to the
// verified context and to the tokens on its root-to-node path; Sec. 3.3
// hands the pruned tree to that single forward pass).  Contract:
// include/dart_verify.h.
//
// Three launches per call:
//   attn_rope_kernel   rotates the tree queries and keys by their position
//                      ids (rotate-half RoPE, fp32, rounded to bf16) into the
//                      workspace; queries are regrouped so the Hq/Hkv query
//                      heads of one kv head are adjacent rows;
//   tree_attn_kernel   flash attention on the tensor cores (tcgen05, TMEM
//                      accumulators, TMA-staged K/V).  A CTA owns 128 query
//                      rows = 128/G tree rows x the G query heads sharing one
//                      kv head, so each K/V tile feeds all G heads.  Its key
//                      tiles are the context tiles (all visible, ragged tail
//                      masked) followed by the tree tiles up to its last row
//                      (ancestors precede their descendants, so later tiles
//                      are invisible), masked by the ancestor bitmask.  Long
//                      key lists are split over `splits` CTAs whose last
//                      finisher merges the partial (max, sum, O) in split
//                      order (deterministic, nobody waits);
//   ancestor mask      (dart_ancestor_mask only) one block per sequence.
// Warp roles of tree_attn_kernel (192 threads): warp 0 TMA producer, warp 1
// TMEM allocator + single-thread MMA issuer, warps 2-5 softmax, thread =
// query row = TMEM lane.  TMEM: two S buffers (128 columns each, so the
// S = Q K^T of tile i+1 overlaps the softmax of tile i) and the O accumulator
// (128 columns).  O stays in TMEM for the whole key range; a row's running
// max is raised (and O, l rescaled through tcgen05.ld/st) only when a tile
// exceeds it by more than 2^8, so P = exp2(s - m) <= 256 and the rescale is
// rare.  Every wait is bounded (status bit on timeout, then drain and exit).
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>
#include <cstring>

#include "../../include/dart.h"
#include "../../include/dart_verify.h"
#include "dart_device.cuh"
#include "dart_kernels.h"

namespace dart {
namespace {

constexpr int kDh = 128;                  // head dimension (two 64-element swizzle columns)
constexpr int kRows = 128;                // query rows per CTA (MMA M)
constexpr int kKeys = 128;                // keys per tile (MMA N of S = QK^T, K of O += PV)
constexpr int kAttnThreads = 192;
constexpr int kSoftThreads = 128;
constexpr int kKvStages = 2;
constexpr int kHalf = kRows * 64 * 2;     // 16 KB: 128 rows x 64 bf16, one 128-byte swizzle column
constexpr int kTileBytes = 2 * kHalf;     // 32 KB: 128 rows x dh bf16
constexpr int kMaxSplits = 16;
constexpr int kTmemCols = 512;            // S0 [0,128), S1 [128,256), O [256,384)
constexpr int kOCol = 256;
constexpr float kRescaleSlack = 8.0f;     // log2 units: P <= 2^8 between rescales
constexpr int kSmemUsed = kTileBytes * (1 + 2 * kKvStages + 1) + 16 * 8 + 4 * 4;
constexpr int kAttnSmem = kSmemUsed + 1024;  // + alignment slack of the 1024-byte swizzle atoms

struct AttnArgs {
    int B, C, Hq, Hkv, G, qpt, nqt, splits, mw, nct;
    float sl2;                // scale * log2(e)
    const int32_t* n_nodes;   // [nseq]
    const uint64_t* mask;     // [nseq][B][mw]
    float* out;               // [nseq][B][Hq][dh]
    float* part_o;            // [blocks][splits][dh][128]
    float2* part_ml;          // [blocks][splits][128] (running max in log2 units, sum)
    int* ticket;              // [blocks], zero on entry
    int* status;
};

struct RopeArgs {
    int nseq, B, Hq, Hkv, G;
    const __nv_bfloat16* q;   // [nseq][B][Hq][dh]
    const __nv_bfloat16* kt;  // [nseq][B][Hkv][dh]
    const int32_t* pos_ids;   // [nseq][B]
    __nv_bfloat16* qr;        // [nseq][Hkv][B][G][dh]
    __nv_bfloat16* kr;        // [nseq][B][Hkv][dh]
    float inv_freq[kDh / 2];
};

// ------------------------------------------------------------ PTX helpers

__device__ __forceinline__ void tma_load_4d(void* dst, const CUtensorMap* map, uint64_t* bar, int x, int y, int z,
                                            int w, uint64_t policy) {
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%0], [%1, {%3, %4, %5, %6}], [%2], %7;" ::"r"(smem_u32(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(x), "r"(y), "r"(z), "r"(w), "l"(policy)
        : "memory");
}

// Descriptor of an MN-major operand written by TMA with 128-byte swizzling:
// 64 MN elements (128 bytes) per row, 8 K rows per 1024-byte atom (stride
// byte offset), the next 64 MN elements `lbo` bytes further (leading byte
// offset).  Used for V (N = head dim contiguous, K = keys).
__device__ __forceinline__ uint64_t sdesc_sw128_mn(uint32_t saddr, uint32_t lbo) {
    uint64_t d = 0;
    d |= static_cast<uint64_t>((saddr >> 4) & 0x3FFFu);
    d |= static_cast<uint64_t>((lbo >> 4) & 0x3FFFu) << 16;
    d |= static_cast<uint64_t>((1024u >> 4) & 0x3FFFu) << 32;
    d |= static_cast<uint64_t>(1u) << 46;
    d |= static_cast<uint64_t>(2u) << 61;
    return d;
}

__device__ __forceinline__ void tmem_st16(uint32_t taddr, const float (&v)[16]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(
            taddr),
        "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])),
        "r"(__float_as_uint(v[3])), "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])),
        "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])), "r"(__float_as_uint(v[8])),
        "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
        "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
        "r"(__float_as_uint(v[15]))
        : "memory");
}
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// Generic-proxy shared-memory writes become visible to the tensor core.
__device__ __forceinline__ void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

__device__ __forceinline__ void attn_timeout(int* status, volatile int* abort) {
    *abort = 1;
    if (status) atomicOr(status, kDevTimeout);
}
__device__ __forceinline__ void attn_drain(uint64_t* bar, uint32_t parity) {
    const unsigned long long t0 = globaltimer_ns();
    while (!mbar_try_wait(bar, parity)) {
        if (globaltimer_ns() - t0 > kWaitLimitNs) return;
    }
}

// A wait whose outcome is the same for every lane of the warp (the
// tcgen05.ld / st that follow are warp-collective).
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort) {
    const bool got = mbar_wait(bar, parity, abort);
    return __all_sync(0xFFFFFFFFu, got);
}

__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<const uint32_t*>(&h);
}

// ------------------------------------------------------------ RoPE pre-pass

__global__ void __launch_bounds__(256) attn_rope_kernel(const RopeArgs a) {
    pdl_trigger();
    pdl_wait();
    constexpr int kPairs = kDh / 4;  // threads per row: two rotation pairs each
    const long long qrows = static_cast<long long>(a.nseq) * a.B * a.Hq;
    const long long rows = qrows + static_cast<long long>(a.nseq) * a.B * a.Hkv;
    for (long long u = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; u < rows * kPairs;
         u += static_cast<long long>(gridDim.x) * blockDim.x) {
        const long long row = u / kPairs;
        const int t = static_cast<int>(u % kPairs) * 2;
        const __nv_bfloat16* src;
        __nv_bfloat16* dst;
        int sb;  // s * B + b
        if (row < qrows) {
            const int h = static_cast<int>(row % a.Hq);
            sb = static_cast<int>(row / a.Hq);
            const int s = sb / a.B, b = sb % a.B, kvh = h / a.G, g = h % a.G;
            src = a.q + row * kDh;
            dst = a.qr + ((((static_cast<long long>(s) * a.Hkv + kvh) * a.B + b) * a.G + g) * kDh);
        } else {
            const long long kr = row - qrows;
            sb = static_cast<int>(kr / a.Hkv);
            src = a.kt + kr * kDh;
            dst = a.kr + kr * kDh;
        }
        const float pos = static_cast<float>(a.pos_ids[sb]);
        const __nv_bfloat162 x1 = *reinterpret_cast<const __nv_bfloat162*>(src + t);
        const __nv_bfloat162 x2 = *reinterpret_cast<const __nv_bfloat162*>(src + t + kDh / 2);
        float s0, c0, s1, c1;
        sincosf(pos * a.inv_freq[t], &s0, &c0);
        sincosf(pos * a.inv_freq[t + 1], &s1, &c1);
        const float a0 = __low2float(x1), a1 = __high2float(x1);
        const float b0 = __low2float(x2), b1 = __high2float(x2);
        *reinterpret_cast<__nv_bfloat162*>(dst + t) = __floats2bfloat162_rn(a0 * c0 - b0 * s0, a1 * c1 - b1 * s1);
        *reinterpret_cast<__nv_bfloat162*>(dst + t + kDh / 2) =
            __floats2bfloat162_rn(b0 * c0 + a0 * s0, b1 * c1 + a1 * s1);
    }
}

// ------------------------------------------------------------ attention

__global__ void __launch_bounds__(kAttnThreads, 1)
    tree_attn_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmKc,
                     const __grid_constant__ CUtensorMap tmVc, const __grid_constant__ CUtensorMap tmKt,
                     const __grid_constant__ CUtensorMap tmVt, const AttnArgs a) {
    extern __shared__ uint8_t attn_smem_raw[];
    pdl_trigger();
    const uint32_t off = (1024u - (smem_u32(attn_smem_raw) & 1023u)) & 1023u;
    uint8_t* sQ = attn_smem_raw + off;
    uint8_t* sKV = sQ + kTileBytes;  // stage st: K at st * 2 * kTileBytes, V right after
    uint8_t* sP = sKV + kKvStages * 2 * kTileBytes;
    uint64_t* bars = reinterpret_cast<uint64_t*>(sP + kTileBytes);
    uint64_t* q_full = bars;
    uint64_t* k_full = bars + 1;     // [2]
    uint64_t* v_full = bars + 3;     // [2]
    uint64_t* kv_empty = bars + 5;   // [2]
    uint64_t* s_full = bars + 7;     // [2]
    uint64_t* s_empty = bars + 9;    // [2]
    uint64_t* p_full = bars + 11;
    uint64_t* pv_done = bars + 12;
    uint64_t* tdown = bars + 13;
    int* misc = reinterpret_cast<int*>(bars + 16);  // [0] TMEM base, [1] abort, [2] last split
    volatile int* abort = &misc[1];

    const int split = blockIdx.x % a.splits;
    const int blk = blockIdx.x / a.splits;
    const int qt = blk % a.nqt;
    const int kvh = (blk / a.nqt) % a.Hkv;
    const int s = blk / (a.nqt * a.Hkv);
    const int q0 = qt * a.qpt;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        mbar_init(q_full, 1);
        for (int i = 0; i < 2; i++) {
            mbar_init(&k_full[i], 1);
            mbar_init(&v_full[i], 1);
            mbar_init(&kv_empty[i], 1);
            mbar_init(&s_full[i], 1);
            mbar_init(&s_empty[i], kSoftThreads);
        }
        mbar_init(p_full, kSoftThreads);
        mbar_init(pv_done, 1);
        mbar_init(tdown, 1);
        misc[1] = 0;
        misc[2] = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(reinterpret_cast<uint32_t*>(&misc[0]), kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = static_cast<uint32_t>(misc[0]);
    pdl_wait();  // rotated queries / keys and the tree arrays come from earlier kernels

    const int nn = min(max(__ldg(a.n_nodes + s), 0), a.B);
    const int qlast = min(q0 + a.qpt, nn) - 1;  // last tree row of this CTA with a query (-1: none)
    const int T = qlast >= 0 ? a.nct + qlast / kKeys + 1 : 0;
    const int j0 = static_cast<int>((static_cast<long long>(split) * T) / a.splits);
    const int nt = static_cast<int>((static_cast<long long>(split + 1) * T) / a.splits) - j0;

    if (warp == 0) {
        // ---------------------------------------------------------- producer
        if (lane == 0 && nt > 0) {
            const uint64_t pol_q = l2_policy_evict_first();
            const uint64_t pol_kv = l2_policy_evict_last();  // re-read by the other query tiles
            const int qrow = ((s * a.Hkv + kvh) * a.B + q0) * a.G;
            mbar_arrive_expect_tx(q_full, kTileBytes);
            tma_load_2d(sQ, &tmQ, q_full, 0, qrow, pol_q);
            tma_load_2d(sQ + kHalf, &tmQ, q_full, 64, qrow, pol_q);
            int issued = 0;
            for (int i = 0; i < nt; i++) {
                const int st = i & 1;
                const uint32_t u = static_cast<uint32_t>(i >> 1);
                if (!mbar_wait(&kv_empty[st], (u & 1u) ^ 1u, abort)) {
                    attn_timeout(a.status, abort);
                    break;
                }
                const int j = j0 + i;
                const bool ctx = j < a.nct;
                const int key0 = (ctx ? j : j - a.nct) * kKeys;
                const CUtensorMap* mk = ctx ? &tmKc : &tmKt;
                const CUtensorMap* mv = ctx ? &tmVc : &tmVt;
                uint8_t* sK = sKV + st * 2 * kTileBytes;
                uint8_t* sV = sK + kTileBytes;
                mbar_arrive_expect_tx(&k_full[st], kTileBytes);
                tma_load_4d(sK, mk, &k_full[st], 0, kvh, key0, s, pol_kv);
                tma_load_4d(sK + kHalf, mk, &k_full[st], 64, kvh, key0, s, pol_kv);
                mbar_arrive_expect_tx(&v_full[st], kTileBytes);
                tma_load_4d(sV, mv, &v_full[st], 0, kvh, key0, s, pol_kv);
                tma_load_4d(sV + kHalf, mv, &v_full[st], 64, kvh, key0, s, pol_kv);
                issued = i + 1;
            }
            if (*abort) {
                // copies still in flight must land before the CTA exits
                attn_drain(q_full, 0);
                for (int i = issued > kKvStages ? issued - kKvStages : 0; i < issued; i++) {
                    attn_drain(&k_full[i & 1], static_cast<uint32_t>(i >> 1) & 1u);
                    attn_drain(&v_full[i & 1], static_cast<uint32_t>(i >> 1) & 1u);
                }
            }
        }
    } else if (warp == 1) {
        // ---------------------------------------------------------- MMA issuer
        if (lane == 0 && nt > 0) {
            constexpr uint32_t idesc_s = idesc_bf16_f32(kRows, kKeys);
            constexpr uint32_t idesc_pv = idesc_bf16_f32(kRows, kDh) | (1u << 16);  // B (= V) MN-major
            const uint32_t q_addr = smem_u32(sQ), p_addr = smem_u32(sP);
            bool ok = mbar_wait(q_full, 0, abort);
            if (!ok) attn_timeout(a.status, abort);
            tc_fence_after();
            auto issue_s = [&](int i) -> bool {
                const int st = i & 1;
                const uint32_t u = static_cast<uint32_t>(i >> 1);
                if (!mbar_wait(&k_full[st], u & 1u, abort) || !mbar_wait(&s_empty[st], (u & 1u) ^ 1u, abort)) {
                    attn_timeout(a.status, abort);
                    return false;
                }
                tc_fence_after();
                const uint32_t k_addr = smem_u32(sKV + st * 2 * kTileBytes);
#pragma unroll
                for (int kk = 0; kk < kDh / 16; kk++) {
                    const uint32_t o = (kk >> 2) * kHalf + (kk & 3) * 32;
                    tc_mma_bf16(tmem + st * kKeys, sdesc_sw128(q_addr + o), sdesc_sw128(k_addr + o), idesc_s,
                                kk > 0 ? 1u : 0u);
                }
                tc_commit(&s_full[st]);
                return true;
            };
            auto issue_pv = [&](int i) -> bool {
                const int st = i & 1;
                if (!mbar_wait(p_full, static_cast<uint32_t>(i) & 1u, abort) ||
                    !mbar_wait(&v_full[st], static_cast<uint32_t>(i >> 1) & 1u, abort)) {
                    attn_timeout(a.status, abort);
                    return false;
                }
                tc_fence_after();
                const uint32_t v_addr = smem_u32(sKV + st * 2 * kTileBytes + kTileBytes);
#pragma unroll
                for (int kk = 0; kk < kKeys / 16; kk++) {
                    const uint32_t o = (kk >> 2) * kHalf + (kk & 3) * 32;
                    tc_mma_bf16(tmem + kOCol, sdesc_sw128(p_addr + o), sdesc_sw128_mn(v_addr + kk * 2048, kHalf),
                                idesc_pv, (i > 0 || kk > 0) ? 1u : 0u);
                }
                tc_commit(&kv_empty[st]);
                tc_commit(pv_done);
                return true;
            };
            if (ok) ok = issue_s(0);
            for (int i = 1; i < nt && ok; i++) {
                ok = issue_s(i);
                if (ok) ok = issue_pv(i - 1);
            }
            if (ok) ok = issue_pv(nt - 1);
            if (!ok) {
                tc_commit(tdown);
                attn_drain(tdown, 0);
            }
        }
    } else {
        // ---------------------------------------------------------- softmax
        const int qd = warp & 3;
        const int r = qd * 32 + lane;          // query row = TMEM lane
        const int b = q0 + r / a.G, g = r % a.G;
        const bool row_ok = b < nn;
        const uint32_t tl = tmem + (static_cast<uint32_t>(qd * 32) << 16);
        uint8_t* prow = sP + r * 128;
        const uint32_t swz = static_cast<uint32_t>(r & 7);
        float m_run = -INFINITY, l = 0.0f;
        bool ok = true;
        for (int i = 0; i < nt; i++) {
            const int j = j0 + i;
            const int st = i & 1;
            const uint32_t u = static_cast<uint32_t>(i >> 1);
            // visible keys of this row in the tile, as two 64-bit words
            uint64_t w0 = 0ull, w1 = 0ull;
            if (row_ok) {
                int kvalid;
                if (j < a.nct) {
                    kvalid = min(kKeys, a.C - j * kKeys);
                    w0 = ~0ull;
                    w1 = ~0ull;
                } else {
                    const int t = j - a.nct;
                    kvalid = min(kKeys, nn - t * kKeys);
                    const uint64_t* mrow = a.mask + (static_cast<size_t>(s) * a.B + b) * a.mw;
                    w0 = __ldg(mrow + 2 * t);
                    w1 = 2 * t + 1 < a.mw ? __ldg(mrow + 2 * t + 1) : 0ull;
                }
                if (kvalid < 64) {
                    w0 &= (1ull << kvalid) - 1ull;
                    w1 = 0ull;
                } else if (kvalid < 128) {
                    w1 &= (1ull << (kvalid - 64)) - 1ull;
                }
            }
            if (!warp_wait(&s_full[st], u & 1u, abort)) {
                attn_timeout(a.status, abort);
                ok = false;
                break;
            }
            tc_fence_after();
            const uint32_t ts = tl + st * kKeys;
            float mx = -INFINITY;
#pragma unroll
            for (int c0 = 0; c0 < kKeys; c0 += 32) {
                float va[16], vb[16];
                tmem_ld16_pair(ts + c0, ts + c0 + 16, va, vb);
                const uint64_t w = c0 < 64 ? w0 : w1;
                const int sh = c0 & 63;
#pragma unroll
                for (int e = 0; e < 16; e++) {
                    if ((w >> (sh + e)) & 1ull) mx = fmaxf(mx, va[e]);
                    if ((w >> (sh + 16 + e)) & 1ull) mx = fmaxf(mx, vb[e]);
                }
            }
            const float mx2 = mx * a.sl2;
            const bool resc = mx2 > m_run + kRescaleSlack;
            const float m_new = resc ? mx2 : m_run;
            const float alpha = resc ? exp2f(m_run - m_new) : 1.0f;
            if (i > 0) {
                // PV of the previous tile must be done before P or O is touched
                if (!warp_wait(pv_done, static_cast<uint32_t>(i - 1) & 1u, abort)) {
                    attn_timeout(a.status, abort);
                    ok = false;
                    break;
                }
                tc_fence_after();
                if (__any_sync(0xFFFFFFFFu, resc)) {
#pragma unroll
                    for (int c0 = 0; c0 < kDh; c0 += 16) {
                        float o[16];
                        tmem_ld16(tl + kOCol + c0, o);
#pragma unroll
                        for (int e = 0; e < 16; e++) o[e] *= alpha;
                        tmem_st16(tl + kOCol + c0, o);
                    }
                    tmem_wait_st();
                }
            }
            l *= alpha;
            m_run = m_new;
            // P = exp2(s * scale * log2 e - m) as bf16 into the swizzled K-major P tile
#pragma unroll
            for (int c0 = 0; c0 < kKeys; c0 += 32) {
                float va[16], vb[16];
                tmem_ld16_pair(ts + c0, ts + c0 + 16, va, vb);
                const uint64_t w = c0 < 64 ? w0 : w1;
                const int sh = c0 & 63;
                uint32_t pk[16];
#pragma unroll
                for (int e = 0; e < 16; e += 2) {
                    const float p0 = ((w >> (sh + e)) & 1ull) ? exp2f(fmaf(va[e], a.sl2, -m_run)) : 0.0f;
                    const float p1 = ((w >> (sh + e + 1)) & 1ull) ? exp2f(fmaf(va[e + 1], a.sl2, -m_run)) : 0.0f;
                    const float p2 = ((w >> (sh + 16 + e)) & 1ull) ? exp2f(fmaf(vb[e], a.sl2, -m_run)) : 0.0f;
                    const float p3 =
                        ((w >> (sh + 16 + e + 1)) & 1ull) ? exp2f(fmaf(vb[e + 1], a.sl2, -m_run)) : 0.0f;
                    pk[e / 2] = pack_bf16(p0, p1);
                    pk[8 + e / 2] = pack_bf16(p2, p3);
                }
                // the sum uses the rounded weights the tensor core multiplies
#pragma unroll
                for (int e = 0; e < 16; e++) {
                    const __nv_bfloat162 h = *reinterpret_cast<const __nv_bfloat162*>(&pk[e]);
                    l += __low2float(h) + __high2float(h);
                }
                // 32 keys = four 16-byte chunks of the 128-byte row of swizzle column c0 / 64
                uint8_t* col = prow + (c0 >> 6) * kHalf;
                const uint32_t ch0 = static_cast<uint32_t>((c0 & 63) >> 3);
#pragma unroll
                for (int q = 0; q < 4; q++) {
                    uint4 v = make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
                    *reinterpret_cast<uint4*>(col + (((ch0 + q) ^ swz) << 4)) = v;
                }
            }
            tc_fence_before();
            mbar_arrive(&s_empty[st]);
            fence_async_smem();
            mbar_arrive(p_full);
        }
        if (ok && nt > 0) {
            if (!warp_wait(pv_done, static_cast<uint32_t>(nt - 1) & 1u, abort)) {
                attn_timeout(a.status, abort);
                ok = false;
            }
            tc_fence_after();
        }
        const int h = kvh * a.G + g;
        if (a.splits == 1) {
            if (ok) {
                float* orow = a.out + ((static_cast<size_t>(s) * a.B + b) * a.Hq + h) * kDh;
                const bool have = nt > 0;
                const float inv = (row_ok && l > 0.0f) ? 1.0f / l : 0.0f;
#pragma unroll
                for (int c0 = 0; c0 < kDh; c0 += 16) {
                    float o[16];
                    if (have) {
                        tmem_ld16(tl + kOCol + c0, o);
                    } else {
#pragma unroll
                        for (int e = 0; e < 16; e++) o[e] = 0.0f;
                    }
                    if (b < a.B) {
#pragma unroll
                        for (int e = 0; e < 16; e += 4)
                            *reinterpret_cast<float4*>(orow + c0 + e) =
                                make_float4(o[e] * inv, o[e + 1] * inv, o[e + 2] * inv, o[e + 3] * inv);
                    }
                }
            }
        } else {
            // partial of this split: (m, l) and O unnormalised, column-major so
            // that a warp's 32 rows are one 128-byte line.  Every softmax warp
            // reaches both named barriers, also after a timeout.
            const size_t pidx = static_cast<size_t>(blk) * a.splits + split;
            a.part_ml[pidx * kRows + r] = make_float2(m_run, (ok && nt > 0) ? l : 0.0f);
            if (ok && nt > 0) {
                float* po = a.part_o + pidx * kDh * kRows + r;
#pragma unroll
                for (int c0 = 0; c0 < kDh; c0 += 16) {
                    float o[16];
                    tmem_ld16(tl + kOCol + c0, o);
#pragma unroll
                    for (int e = 0; e < 16; e++) po[(c0 + e) * kRows] = o[e];
                }
            }
            __threadfence();
            named_bar_sync(kEpiBarrier, kSoftThreads);
            if (r == 0) {
                const int tk = atomicAdd(&a.ticket[blk], 1);
                misc[2] = tk == a.splits - 1;
                if (tk == a.splits - 1) a.ticket[blk] = 0;
            }
            named_bar_sync(kEpiBarrier, kSoftThreads);
            if (misc[2]) {
                __threadfence();
                // merge the splits in order: O = sum_p 2^(m_p - M) O_p / sum_p 2^(m_p - M) l_p
                const size_t p0 = static_cast<size_t>(blk) * a.splits;
                float M = -INFINITY;
                for (int p = 0; p < a.splits; p++) {
                    const float2 ml = __ldcg(a.part_ml + (p0 + p) * kRows + r);
                    if (ml.y > 0.0f) M = fmaxf(M, ml.x);
                }
                float wsum = 0.0f;
                float wp[kMaxSplits];
#pragma unroll
                for (int p = 0; p < kMaxSplits; p++) {
                    wp[p] = 0.0f;
                    if (p < a.splits) {
                        const float2 ml = __ldcg(a.part_ml + (p0 + p) * kRows + r);
                        if (ml.y > 0.0f) {
                            wp[p] = exp2f(ml.x - M);
                            wsum += wp[p] * ml.y;
                        }
                    }
                }
                const float inv = (row_ok && wsum > 0.0f) ? 1.0f / wsum : 0.0f;
                if (b < a.B) {
                    float* orow = a.out + ((static_cast<size_t>(s) * a.B + b) * a.Hq + h) * kDh;
                    for (int c0 = 0; c0 < kDh; c0 += 4) {
                        float o[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
                        for (int p = 0; p < kMaxSplits; p++) {
                            if (p < a.splits && wp[p] != 0.0f) {
                                const float* po = a.part_o + (p0 + p) * kDh * kRows + r;
#pragma unroll
                                for (int e = 0; e < 4; e++) o[e] += wp[p] * __ldcg(po + (c0 + e) * kRows);
                            }
                        }
                        *reinterpret_cast<float4*>(orow + c0) =
                            make_float4(o[0] * inv, o[1] * inv, o[2] * inv, o[3] * inv);
                    }
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

// ------------------------------------------------------------ ancestor mask

constexpr int kMaskThreads = 1024;

__global__ void __launch_bounds__(kMaskThreads) ancestor_mask_kernel(const int32_t* parents, const int32_t* n_nodes,
                                                                      int B, uint64_t* mask) {
    pdl_trigger();
    pdl_wait();
    const int s = blockIdx.x, mw = (B + 63) / 64;
    const int nn = min(max(n_nodes[s], 0), B);
    const int32_t* par = parents + static_cast<size_t>(s) * B;
    for (int q = threadIdx.x; q < B * mw; q += kMaskThreads) {
        const int i = q / mw, wd = q % mw;
        uint64_t word = 0ull;
        if (i < nn) {
            int j = i;
            for (int steps = 0; steps <= i && j >= 0; steps++) {
                if ((j >> 6) == wd) word |= 1ull << (j & 63);
                const int pj = par[j];
                if (pj < -1 || pj >= j) break;
                j = pj;
            }
        }
        mask[(static_cast<size_t>(s) * B + i) * mw + wd] = word;
    }
}

// ------------------------------------------------------------ host helpers

struct Plan {
    int G, qpt, nqt, blocks, splits, mw, nct;
    size_t off_qr, off_kr, off_po, off_ml, off_ticket, total;
};

size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

bool valid_cfg(const dart_attn_config* c) {
    if (!c) return false;
    if (c->nseq < 1 || c->B < 1 || c->B > 1024 || c->C < 0 || c->Hkv < 1 || c->Hq < c->Hkv) return false;
    if (c->Hq % c->Hkv != 0) return false;
    const int G = c->Hq / c->Hkv;
    if (G != 1 && G != 2 && G != 4 && G != 8 && G != 16) return false;
    if (c->dh != kDh) return false;
    if (!(c->rope_theta > 1.0f) || !std::isfinite(c->rope_theta)) return false;
    if (!(c->scale > 0.0f) || !std::isfinite(c->scale)) return false;
    // TMA coordinates and element counts stay in int range
    if (static_cast<long long>(c->nseq) * c->Hq * c->B > (1ll << 30)) return false;
    if (static_cast<long long>(c->C) * c->Hkv * kDh > (1ll << 40)) return false;
    return true;
}

int sm_count() {
    int dev = 0, n = 148;
    if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    return n > 0 ? n : 148;
}

// Splits of the key list: the smallest modelled time ceil(CTAs / SMs) waves
// x tiles per split, plus one tile for the merge when split.
int pick_splits(int blocks, int max_tiles, int nsm) {
    int best = 1;
    long long best_cost = -1;
    for (int sp = 1; sp <= kMaxSplits; sp++) {
        if (sp > 1 && (max_tiles + sp - 1) / sp < 2) break;
        const long long waves = (static_cast<long long>(blocks) * sp + nsm - 1) / nsm;
        const long long cost = waves * ((max_tiles + sp - 1) / sp) + (sp > 1 ? 1 : 0);
        if (best_cost < 0 || cost < best_cost) {
            best_cost = cost;
            best = sp;
        }
    }
    return best;
}

Plan make_plan(const dart_attn_config* c, int nsm) {
    Plan p;
    p.G = c->Hq / c->Hkv;
    p.qpt = kRows / p.G;
    p.nqt = (c->B + p.qpt - 1) / p.qpt;
    p.blocks = c->nseq * c->Hkv * p.nqt;
    p.mw = (c->B + 63) / 64;
    p.nct = (c->C + kKeys - 1) / kKeys;
    p.splits = pick_splits(p.blocks, p.nct + (c->B + kKeys - 1) / kKeys, nsm);
    const size_t qr = static_cast<size_t>(c->nseq) * c->B * c->Hq * kDh * 2;
    const size_t kr = static_cast<size_t>(c->nseq) * c->B * c->Hkv * kDh * 2;
    const size_t po = p.splits > 1 ? static_cast<size_t>(p.blocks) * p.splits * kDh * kRows * 4 : 0;
    const size_t ml = p.splits > 1 ? static_cast<size_t>(p.blocks) * p.splits * kRows * 8 : 0;
    const size_t tk = p.splits > 1 ? static_cast<size_t>(p.blocks) * 4 : 0;
    p.off_qr = 0;
    p.off_kr = align256(p.off_qr + qr);
    p.off_po = align256(p.off_kr + kr);
    p.off_ml = align256(p.off_po + po);
    p.off_ticket = align256(p.off_ml + ml);
    p.total = align256(p.off_ticket + tk);
    return p;
}

bool encode_2d(CUtensorMap* m, const void* base, uint64_t rows) {
    EncodeTiledFn fn = tensor_map_encoder();
    if (!fn) return false;
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(kDh), rows};
    cuuint64_t strides[1] = {kDh * 2};
    cuuint32_t box[2] = {64, kRows};
    cuuint32_t estr[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// [nseq][len][Hkv][dh] bf16 with a (64, 1, 128 keys, 1) box.
bool encode_kv(CUtensorMap* m, const void* base, int nseq, int len, int Hkv) {
    EncodeTiledFn fn = tensor_map_encoder();
    if (!fn) return false;
    cuuint64_t dims[4] = {static_cast<cuuint64_t>(kDh), static_cast<cuuint64_t>(Hkv), static_cast<cuuint64_t>(len),
                          static_cast<cuuint64_t>(nseq)};
    cuuint64_t strides[3] = {static_cast<cuuint64_t>(kDh) * 2, static_cast<cuuint64_t>(Hkv) * kDh * 2,
                             static_cast<cuuint64_t>(len) * Hkv * kDh * 2};
    cuuint32_t box[4] = {64, 1, kKeys, 1};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool al16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace
}  // namespace dart

using namespace dart;

extern "C" {

size_t dart_tree_attention_workspace(const dart_attn_config* cfg) {
    if (!valid_cfg(cfg)) return 0;
    return make_plan(cfg, sm_count()).total;
}

int dart_tree_attention(const dart_attn_config* cfg, const void* q, const void* k_tree, const void* v_tree,
                        const void* k_ctx, const void* v_ctx, const int32_t* pos_ids, const uint64_t* mask,
                        const int32_t* n_nodes, float* out, void* workspace, size_t workspace_bytes, int* status,
                        void* stream) {
    if (!valid_cfg(cfg)) return DART_ERR_INVALID;
    const dart_attn_config& c = *cfg;
    if (!q || !k_tree || !v_tree || !pos_ids || !mask || !n_nodes || !out || !workspace) return DART_ERR_INVALID;
    if (c.C > 0 && (!k_ctx || !v_ctx)) return DART_ERR_INVALID;
    if (!al16(q) || !al16(k_tree) || !al16(v_tree) || !al16(out) || !al16(mask) || !al16(pos_ids) ||
        !al16(n_nodes) || (reinterpret_cast<uintptr_t>(workspace) & 255u))
        return DART_ERR_INVALID;
    if (c.C > 0 && (!al16(k_ctx) || !al16(v_ctx))) return DART_ERR_INVALID;
    if (status && !al16(status)) return DART_ERR_INVALID;
    int dev = 0, major = 0, minor = 0, optin = 0, nsm = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return DART_ERR_CUDA;
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
    cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
    if (major != 10 || minor != 3 || optin < kAttnSmem) return DART_ERR_UNSUPPORTED;
    const Plan p = make_plan(cfg, nsm > 0 ? nsm : 148);
    if (workspace_bytes < p.total) return DART_ERR_INVALID;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    uint8_t* ws = static_cast<uint8_t*>(workspace);
    __nv_bfloat16* qr = reinterpret_cast<__nv_bfloat16*>(ws + p.off_qr);
    __nv_bfloat16* kr = reinterpret_cast<__nv_bfloat16*>(ws + p.off_kr);

    CUtensorMap tmQ, tmKc, tmVc, tmKt, tmVt;
    if (!encode_2d(&tmQ, qr, static_cast<uint64_t>(c.nseq) * c.Hkv * c.B * p.G)) return DART_ERR_CUDA;
    if (!encode_kv(&tmKt, kr, c.nseq, c.B, c.Hkv) || !encode_kv(&tmVt, v_tree, c.nseq, c.B, c.Hkv))
        return DART_ERR_CUDA;
    if (c.C > 0) {
        if (!encode_kv(&tmKc, k_ctx, c.nseq, c.C, c.Hkv) || !encode_kv(&tmVc, v_ctx, c.nseq, c.C, c.Hkv))
            return DART_ERR_CUDA;
    } else {
        tmKc = tmKt;  // never read: no context tiles
        tmVc = tmVt;
    }

    RopeArgs ra;
    std::memset(&ra, 0, sizeof ra);
    ra.nseq = c.nseq;
    ra.B = c.B;
    ra.Hq = c.Hq;
    ra.Hkv = c.Hkv;
    ra.G = p.G;
    ra.q = static_cast<const __nv_bfloat16*>(q);
    ra.kt = static_cast<const __nv_bfloat16*>(k_tree);
    ra.pos_ids = pos_ids;
    ra.qr = qr;
    ra.kr = kr;
    for (int t = 0; t < kDh / 2; t++)
        ra.inv_freq[t] = static_cast<float>(std::pow(static_cast<double>(c.rope_theta), -2.0 * t / kDh));

    AttnArgs aa;
    std::memset(&aa, 0, sizeof aa);
    aa.B = c.B;
    aa.C = c.C;
    aa.Hq = c.Hq;
    aa.Hkv = c.Hkv;
    aa.G = p.G;
    aa.qpt = p.qpt;
    aa.nqt = p.nqt;
    aa.splits = p.splits;
    aa.mw = p.mw;
    aa.nct = p.nct;
    aa.sl2 = static_cast<float>(static_cast<double>(c.scale) * 1.4426950408889634);
    aa.n_nodes = n_nodes;
    aa.mask = mask;
    aa.out = out;
    aa.part_o = p.splits > 1 ? reinterpret_cast<float*>(ws + p.off_po) : nullptr;
    aa.part_ml = p.splits > 1 ? reinterpret_cast<float2*>(ws + p.off_ml) : nullptr;
    aa.ticket = p.splits > 1 ? reinterpret_cast<int*>(ws + p.off_ticket) : nullptr;
    aa.status = status;

    if (p.splits > 1 && cudaMemsetAsync(aa.ticket, 0, static_cast<size_t>(p.blocks) * 4, st) != cudaSuccess)
        return DART_ERR_CUDA;
    const long long rope_threads = static_cast<long long>(c.nseq) * c.B * (c.Hq + c.Hkv) * (kDh / 4);
    const int rope_blocks = static_cast<int>(std::min<long long>((rope_threads + 255) / 256, 8LL * (nsm > 0 ? nsm : 148)));
    if (launch_pdl(attn_rope_kernel, dim3(rope_blocks), dim3(256), 0, st, ra) != cudaSuccess) return DART_ERR_CUDA;
    if (cudaFuncSetAttribute(tree_attn_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kAttnSmem) !=
        cudaSuccess)
        return DART_ERR_CUDA;
    if (launch_pdl(tree_attn_kernel, dim3(p.blocks * p.splits), dim3(kAttnThreads), kAttnSmem, st, tmQ, tmKc, tmVc,
                   tmKt, tmVt, aa) != cudaSuccess)
        return DART_ERR_CUDA;
    return DART_OK;
}

int dart_ancestor_mask(const int32_t* parents, const int32_t* n_nodes, int nseq, int B, uint64_t* mask,
                       void* stream) {
    if (!parents || !n_nodes || !mask || nseq < 1 || B < 1 || B > 1024) return DART_ERR_INVALID;
    if (reinterpret_cast<uintptr_t>(mask) & 7u) return DART_ERR_INVALID;
    if (launch_pdl(ancestor_mask_kernel, dim3(nseq), dim3(kMaskThreads), 0, static_cast<cudaStream_t>(stream),
                   parents, n_nodes, B, mask) != cudaSuccess)
        return DART_ERR_CUDA;
    return DART_OK;
}

}  // extern "C"
