// Tree-attention verification consumer of the emitted draft tree (Sec. 3.3,
// "Tree Verification and DDTree": every flattened tree node attends to the
// verified context and to the tokens on its root-to-node path; Sec. 4.3
// hands the pruned tree to that single forward pass).  Contract:
// include/dart_verify.h.
//
// Two launches per call:
//   attn_prep_kernel   the RoPE (cos, sin) table of every tree position and
//                      the rotated tree keys (rotate-half RoPE in fp32,
//                      rounded to bf16) in the workspace;
//   tree_attn_kernel   flash attention on the tensor cores (tcgen05, TMEM
//                      operands and accumulators, TMA-staged K/V).  A CTA
//                      owns 128 query rows = 128/G tree rows x the G query
//                      heads sharing one kv head, so each K/V tile feeds all
//                      G heads.  Its key tiles are the context tiles (all
//                      visible, ragged tail masked) followed by the tree
//                      tiles up to its last row (ancestors precede their
//                      descendants, so later tiles are invisible), masked by
//                      the ancestor bitmask.  When there are fewer (sequence,
//                      kv head, query tile) blocks than SMs, the key list is
//                      split over a thread-block cluster of up to 4 CTAs
//                      that merge their partial (max, sum, O) over
//                      distributed shared memory, in rank order;
// and dart_ancestor_mask's own kernel, one block per sequence.
// tree_attn_kernel, 320 threads: warp 0 TMA producer (K ring 3 stages, V ring
// 3 stages), warp 1 TMEM allocator + single-thread MMA issuer, warps 2-9 two
// softmax warpgroups; thread = query row = TMEM lane, warpgroup wg owns key
// columns and O columns [64 wg, 64 wg + 64) of the rows, the pair of warps of
// a lane quarter exchanging row max and row sum through shared memory.
// TMEM (512 columns): S [0,128), O [128,256), P double buffer [256,384), the
// rotated query tile [384,448).  S = Q K^T and O += P V both take A from
// TMEM (K K-major, V MN-major from shared memory); the softmax reads S into
// registers at once, which frees it for the next tile's S while it works.
// O stays in TMEM for the whole key range; a row's running max is raised
// (and O, l rescaled through tcgen05.ld/st) only when a tile exceeds it by
// more than 2^8, so P = exp2(s - m) <= 256 and the rescale is rare.  Every
// wait is bounded (status bit on timeout, then drain and exit).
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <atomic>
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
constexpr int kSoftThreads = 256;             // two softmax warpgroups: key / O columns [0,64) and [64,128)
constexpr int kAttnThreads = 64 + kSoftThreads;
constexpr int kPairBarrier0 = 2;             // named barriers 2..5: the two warps of one TMEM lane quarter
constexpr int kKStages = 3;                  // K ring: the S MMA needs K two tiles ahead of its load
constexpr int kVStages = 3;
constexpr int kHalf = kRows * 64 * 2;     // 16 KB: 128 rows x 64 bf16, one 128-byte swizzle column
constexpr int kTileBytes = 2 * kHalf;     // 32 KB: 128 rows x dh bf16
constexpr int kMaxSplits = 4;                // cluster size: clusters of 4 fit a GPC in one wave beside each other
constexpr int kTmemCols = 512;            // S [0,128), O [128,256), P0 [256,320), P1 [320,384), Q [384,448)
constexpr int kSCol = 0;
constexpr int kOCol = 128;
constexpr int kPCol = 256;                // P tiles: 128 keys as 64 columns of bf16 pairs
constexpr int kQCol = 384;                // rotated query tile: dh = 128 as 64 columns of bf16 pairs
constexpr float kRescaleSlack = 8.0f;     // log2 units: P <= 2^8 between rescales
constexpr int kNumBars = 1 + 2 * kKStages + 2 * kVStages + 2 + 5;
constexpr int kSmemUsed = kTileBytes * (1 + kKStages + kVStages) + kNumBars * 8 + 4 * 4 + 2 * 128 * 4 + 8 * 4;  // Q, K/V rings, barriers, exchange
constexpr int kAttnSmem = kSmemUsed + 1024;  // + alignment slack of the 1024-byte swizzle atoms

struct AttnArgs {
    int B, C, Hq, Hkv, G, qpt, nqt, splits, mw, nct;
    float sl2;                // scale * log2(e)
    const float2* cs;         // [nseq][B][dh/2] RoPE (cos, sin) of the tree positions
    const int32_t* n_nodes;   // [nseq]
    const uint64_t* mask;     // [nseq][B][mw]
    float* out;               // [nseq][B][Hq][dh]
    int* status;
};

struct PrepArgs {
    int nseq, B, Hkv;
    const __nv_bfloat16* kt;  // [nseq][B][Hkv][dh]
    const int32_t* pos_ids;   // [nseq][B]
    __nv_bfloat16* kr;        // [nseq][B][Hkv][dh] rotated tree keys
    float2* cs;               // [nseq][B][dh/2] (cos, sin) of every tree position and frequency
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

// D[tmem] (+)= A[tmem] * B[smem], bf16 inputs, fp32 accumulation (A: lane =
// row, K along columns as bf16 pairs).
__device__ __forceinline__ void tc_mma_bf16_ts(uint32_t tmem_d, uint32_t tmem_a, uint64_t bdesc, uint32_t idesc,
                                               uint32_t accumulate) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
        " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}\n" ::"r"(tmem_d),
        "r"(tmem_a), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// 16 consecutive 32-bit TMEM columns of this thread's lane from registers.
__device__ __forceinline__ void tmem_st16u(uint32_t taddr, const uint32_t (&v)[16]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(
            taddr),
        "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]), "r"(v[9]),
        "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15])
        : "memory");
}

// 32 consecutive 32-bit TMEM columns of this thread's lane from registers.
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&v)[32]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
        "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
        "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]), "r"(v[9]),
        "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15]), "r"(v[16]), "r"(v[17]), "r"(v[18]),
        "r"(v[19]), "r"(v[20]), "r"(v[21]), "r"(v[22]), "r"(v[23]), "r"(v[24]), "r"(v[25]), "r"(v[26]), "r"(v[27]),
        "r"(v[28]), "r"(v[29]), "r"(v[30]), "r"(v[31])
        : "memory");
}

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

// Stores into the shared memory of cluster CTA `rank` at the offset of the
// local shared address `local` (distributed shared memory).
__device__ __forceinline__ void st_cluster_f32x4(uint32_t local, int rank, float x, float y, float z, float w) {
    uint32_t remote;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(local), "r"(rank));
    asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(remote), "f"(x), "f"(y), "f"(z), "f"(w)
                 : "memory");
}
__device__ __forceinline__ void st_cluster_f32x2(uint32_t local, int rank, float x, float y) {
    uint32_t remote;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(local), "r"(rank));
    asm volatile("st.shared::cluster.v2.f32 [%0], {%1, %2};" ::"r"(remote), "f"(x), "f"(y) : "memory");
}

// Column slice [slice_lo(j), slice_lo(j + 1)) merged by cluster CTA j of
// `splits` (multiples of 4 columns), and the padded row stride (floats) of a
// received slice: an odd number of 16-byte units.
__device__ __forceinline__ int slice_lo(int j, int splits) { return 4 * ((j * (kDh / 4)) / splits); }
__device__ __forceinline__ int slice_stride(int ncol) { return ((ncol / 4) & 1) ? ncol : ncol + 4; }

__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<const uint32_t*>(&h);
}

// ------------------------------------------------------------ RoPE pre-pass

// sin and cos of x (|x| up to ~1e5): Cody-Waite reduction by 2*pi split
// into two floats (the high part exactly representable, so k * hi is exact
// inside the fma), then the hardware approximations on [-pi, pi] (absolute
// error ~2^-21, far below the bf16 rounding of the rotated values).
__device__ __forceinline__ void sincos_reduced(float x, float* sn, float* cs) {
    constexpr float kInv2Pi = 0.159154943091895336f;
    constexpr float k2PiHi = 6.28318548202514648f;  // float(2 pi)
    constexpr float k2PiLo = -1.74845560e-7f;       // 2 pi - k2PiHi
    const float k = rintf(x * kInv2Pi);
    float r = fmaf(-k, k2PiHi, x);
    r = fmaf(-k, k2PiLo, r);
    __sincosf(r, sn, cs);
}

// One warp per tree key row (s, b, kv head) -- every row's loads in flight at
// once: the row is rotated into kr (two of the 64 frequencies per lane), and
// the kv-head-0 warp of (s, b) writes the (cos, sin) of its position to the
// table the attention kernel rotates its queries with.
__global__ void __launch_bounds__(256) attn_prep_kernel(const PrepArgs a) {
    pdl_trigger();
    pdl_wait();
    const int lane = threadIdx.x & 31, t = lane * 2;
    const int rows = a.nseq * a.B * a.Hkv;
    const int wstride = gridDim.x * (blockDim.x >> 5);
    for (int row = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); row < rows; row += wstride) {
        const int sb = row / a.Hkv;
        const size_t off = static_cast<size_t>(row) * kDh;
        const __nv_bfloat162 x1 = *reinterpret_cast<const __nv_bfloat162*>(a.kt + off + t);
        const __nv_bfloat162 x2 = *reinterpret_cast<const __nv_bfloat162*>(a.kt + off + t + kDh / 2);
        const float pos = static_cast<float>(__ldg(a.pos_ids + sb));
        float s0, c0, s1, c1;
        sincos_reduced(pos * a.inv_freq[t], &s0, &c0);
        sincos_reduced(pos * a.inv_freq[t + 1], &s1, &c1);
        if (row % a.Hkv == 0)
            *reinterpret_cast<float4*>(a.cs + static_cast<size_t>(sb) * (kDh / 2) + t) = make_float4(c0, s0, c1, s1);
        const float a0 = __low2float(x1), a1 = __high2float(x1);
        const float b0 = __low2float(x2), b1 = __high2float(x2);
        *reinterpret_cast<__nv_bfloat162*>(a.kr + off + t) = __floats2bfloat162_rn(a0 * c0 - b0 * s0, a1 * c1 - b1 * s1);
        *reinterpret_cast<__nv_bfloat162*>(a.kr + off + t + kDh / 2) =
            __floats2bfloat162_rn(b0 * c0 + a0 * s0, b1 * c1 + a1 * s1);
    }
}

// ------------------------------------------------------------ attention

// 64 consecutive 32-bit TMEM columns of this thread's lane into registers
// (two x32 loads, one wait; the registers are tied to the wait so no use can
// move above it).
__device__ __forceinline__ void tmem_ld64(uint32_t taddr, float (&v)[64]) {
    uint32_t r[64];
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
                 : "r"(taddr + 0));
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
                 : "=r"(r[32]), "=r"(r[33]), "=r"(r[34]), "=r"(r[35]), "=r"(r[36]), "=r"(r[37]), "=r"(r[38]), "=r"(r[39]), "=r"(r[40]), "=r"(r[41]), "=r"(r[42]), "=r"(r[43]), "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]), "=r"(r[48]), "=r"(r[49]), "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]), "=r"(r[55]), "=r"(r[56]), "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]), "=r"(r[61]), "=r"(r[62]), "=r"(r[63])
                 : "r"(taddr + 32));
    asm volatile("tcgen05.wait::ld.sync.aligned;"
                 : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]), "+r"(r[14]), "+r"(r[15]), "+r"(r[16]), "+r"(r[17]), "+r"(r[18]), "+r"(r[19]), "+r"(r[20]), "+r"(r[21]), "+r"(r[22]), "+r"(r[23]), "+r"(r[24]), "+r"(r[25]), "+r"(r[26]), "+r"(r[27]), "+r"(r[28]), "+r"(r[29]), "+r"(r[30]), "+r"(r[31]), "+r"(r[32]), "+r"(r[33]), "+r"(r[34]), "+r"(r[35]), "+r"(r[36]), "+r"(r[37]), "+r"(r[38]), "+r"(r[39]), "+r"(r[40]), "+r"(r[41]), "+r"(r[42]), "+r"(r[43]), "+r"(r[44]), "+r"(r[45]), "+r"(r[46]), "+r"(r[47]), "+r"(r[48]), "+r"(r[49]), "+r"(r[50]), "+r"(r[51]), "+r"(r[52]), "+r"(r[53]), "+r"(r[54]), "+r"(r[55]), "+r"(r[56]), "+r"(r[57]), "+r"(r[58]), "+r"(r[59]), "+r"(r[60]), "+r"(r[61]), "+r"(r[62]), "+r"(r[63])
                 :
                 : "memory");
#pragma unroll
    for (int k = 0; k < 64; k++) v[k] = __uint_as_float(r[k]);
}

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__global__ void __launch_bounds__(kAttnThreads, 1)
    tree_attn_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmKc,
                     const __grid_constant__ CUtensorMap tmVc, const __grid_constant__ CUtensorMap tmKt,
                     const __grid_constant__ CUtensorMap tmVt, const AttnArgs a) {
    extern __shared__ uint8_t attn_smem_raw[];
    pdl_trigger();
    const uint32_t off = (1024u - (smem_u32(attn_smem_raw) & 1023u)) & 1023u;
    uint8_t* sQ = attn_smem_raw + off;
    uint8_t* sK = sQ + kTileBytes;                    // [kKStages] K stages
    uint8_t* sV = sK + kKStages * kTileBytes;         // [kVStages] V stages
    uint64_t* bars = reinterpret_cast<uint64_t*>(sV + kVStages * kTileBytes);
    uint64_t* q_full = bars;
    uint64_t* k_full = bars + 1;                      // [kKStages]
    uint64_t* k_empty = k_full + kKStages;            // [kKStages] S of the stage's tile done
    uint64_t* v_full = k_empty + kKStages;            // [kVStages]
    uint64_t* v_empty = v_full + kVStages;            // [kVStages] PV of the stage's tile done
    uint64_t* s_full = v_empty + kVStages;
    uint64_t* s_empty = s_full + 1;                   // softmax has S in registers
    uint64_t* p_full = s_empty + 1;
    uint64_t* pv_done = p_full + 1;                   // [2] PV of a tile using P buffer b done
    uint64_t* tdown = pv_done + 2;
    uint64_t* q_ready = tdown + 1;                    // queries rotated in place
    int* misc = reinterpret_cast<int*>(bars + kNumBars);  // [0] TMEM base, [1] abort
    volatile int* abort = &misc[1];

    // cluster of `splits` CTAs = one (sequence, kv head, query tile); the
    // cluster rank is the key-range split
    const int split = a.splits > 1 ? static_cast<int>(cluster_ctarank()) : 0;
    const int blk = blockIdx.x / a.splits;
    const int qt = blk % a.nqt;
    const int kvh = (blk / a.nqt) % a.Hkv;
    const int s = blk / (a.nqt * a.Hkv);
    const int q0 = qt * a.qpt;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        mbar_init(q_full, 1);
        for (int i = 0; i < kKStages; i++) {
            mbar_init(&k_full[i], 1);
            mbar_init(&k_empty[i], 1);
        }
        for (int i = 0; i < kVStages; i++) {
            mbar_init(&v_full[i], 1);
            mbar_init(&v_empty[i], 1);
        }
        mbar_init(s_full, 1);
        mbar_init(s_empty, kSoftThreads);
        mbar_init(p_full, kSoftThreads);
        mbar_init(&pv_done[0], 1);
        mbar_init(&pv_done[1], 1);
        mbar_init(tdown, 1);
        mbar_init(q_ready, kSoftThreads);
        misc[1] = 0;
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
    pdl_wait();  // the key table, rotated keys and the tree arrays come from earlier kernels

    const int nn = min(max(__ldg(a.n_nodes + s), 0), a.B);
    const int qlast = min(q0 + a.qpt, nn) - 1;  // last tree row of this CTA with a query (-1: none)
    const int T = qlast >= 0 ? a.nct + qlast / kKeys + 1 : 0;
    const int j0 = (split * T) / a.splits;
    const int nt = ((split + 1) * T) / a.splits - j0;

    // softmax state (warps 2-9), kept for the epilogue.  Warps w and w + 4
    // share TMEM lane quarter w % 4 (the same 32 query rows); warpgroup wg
    // handles key columns and O columns [64 wg, 64 wg + 64).
    const int qd = warp & 3;
    const int wg = warp >= 2 ? (warp - 2) >> 2 : 0;
    const int cb = wg * 64;
    const int r = qd * 32 + lane;  // query row = TMEM lane
    const int b = q0 + r / a.G, g = r % a.G;
    const bool row_ok = b < nn;
    const uint32_t tl = tmem + (static_cast<uint32_t>(qd * 32) << 16);
    float* xch = reinterpret_cast<float*>(misc + 4);  // [2][128] row max / sum exchange of the two warpgroups
    int* xok = misc + 4 + 2 * kRows;                   // [2][4] per-warp "no wait failed" exchange
    float m_run = -INFINITY, l = 0.0f;
    bool ok = true;

    if (warp == 0) {
        // ---------------------------------------------------------- producer
        if (lane == 0 && nt > 0) {
            const uint64_t pol_q = l2_policy_evict_first();
            const uint64_t pol_kv = l2_policy_evict_last();  // re-read by the other query tiles
            // rows (tree row q0 + r / G, head kvh * G + r % G)
            mbar_arrive_expect_tx(q_full, kTileBytes);
            tma_load_4d(sQ, &tmQ, q_full, 0, kvh * a.G, q0, s, pol_q);
            tma_load_4d(sQ + kHalf, &tmQ, q_full, 64, kvh * a.G, q0, s, pol_q);
            // K runs up to kKStages tiles ahead, V up to kVStages: issue
            // whichever is due, K first
            int kdone = 0, vdone = 0;
            while ((kdone < nt || vdone < nt) && !*abort) {
                const bool do_k = kdone < nt && kdone < vdone + kKStages;
                const int i = do_k ? kdone : vdone;
                const int j = j0 + i;
                const bool ctx = j < a.nct;
                const int key0 = (ctx ? j : j - a.nct) * kKeys;
                if (do_k) {
                    const int st = i % kKStages;
                    if (!mbar_wait(&k_empty[st], (static_cast<uint32_t>(i / kKStages) & 1u) ^ 1u, abort)) {
                        attn_timeout(a.status, abort);
                        break;
                    }
                    uint8_t* dk = sK + st * kTileBytes;
                    mbar_arrive_expect_tx(&k_full[st], kTileBytes);
                    tma_load_4d(dk, ctx ? &tmKc : &tmKt, &k_full[st], 0, kvh, key0, s, pol_kv);
                    tma_load_4d(dk + kHalf, ctx ? &tmKc : &tmKt, &k_full[st], 64, kvh, key0, s, pol_kv);
                    kdone++;
                } else {
                    const int st = i % kVStages;
                    if (!mbar_wait(&v_empty[st], (static_cast<uint32_t>(i / kVStages) & 1u) ^ 1u, abort)) {
                        attn_timeout(a.status, abort);
                        break;
                    }
                    uint8_t* dv = sV + st * kTileBytes;
                    mbar_arrive_expect_tx(&v_full[st], kTileBytes);
                    tma_load_4d(dv, ctx ? &tmVc : &tmVt, &v_full[st], 0, kvh, key0, s, pol_kv);
                    tma_load_4d(dv + kHalf, ctx ? &tmVc : &tmVt, &v_full[st], 64, kvh, key0, s, pol_kv);
                    vdone++;
                }
            }
            if (*abort) {
                // copies still in flight must land before the CTA exits
                attn_drain(q_full, 0);
                for (int i = kdone > kKStages ? kdone - kKStages : 0; i < kdone; i++)
                    attn_drain(&k_full[i % kKStages], static_cast<uint32_t>(i / kKStages) & 1u);
                for (int i = vdone > kVStages ? vdone - kVStages : 0; i < vdone; i++)
                    attn_drain(&v_full[i % kVStages], static_cast<uint32_t>(i / kVStages) & 1u);
            }
        }
    } else if (warp == 1) {
        // ---------------------------------------------------------- MMA issuer
        // Q (rotated) and P are tensor-memory operands, K and V come from the
        // shared-memory rings.  Order: S(0); then per tile i: S(i+1) once
        // softmax(i) holds S(i) in registers (it runs during softmax(i)),
        // PV(i) once P(i) is written (P is double-buffered).
        if (lane == 0 && nt > 0) {
            constexpr uint32_t idesc_s = idesc_bf16_f32(kRows, kKeys);
            constexpr uint32_t idesc_pv = idesc_bf16_f32(kRows, kDh) | (1u << 16);  // B (= V) MN-major
            bool mok = mbar_wait(q_ready, 0, abort);
            auto issue_s = [&](int i) -> bool {
                const int st = i % kKStages;
                // the S columns were last read by softmax(i - 1)
                if (!mbar_wait(&k_full[st], static_cast<uint32_t>(i / kKStages) & 1u, abort) ||
                    (i > 0 && !mbar_wait(s_empty, static_cast<uint32_t>(i - 1) & 1u, abort)))
                    return false;
                tc_fence_after();
                const uint32_t k_addr = smem_u32(sK + st * kTileBytes);
#pragma unroll
                for (int kk = 0; kk < kDh / 16; kk++) {
                    const uint32_t o = (kk >> 2) * kHalf + (kk & 3) * 32;
                    tc_mma_bf16_ts(tmem + kSCol, tmem + kQCol + kk * 8, sdesc_sw128(k_addr + o), idesc_s,
                                   kk > 0 ? 1u : 0u);
                }
                tc_commit(s_full);
                tc_commit(&k_empty[st]);
                return true;
            };
            if (mok) tc_fence_after();
            if (mok) mok = issue_s(0);
            for (int i = 0; i < nt && mok; i++) {
                if (i + 1 < nt && !issue_s(i + 1)) {
                    mok = false;
                    break;
                }
                const int st = i % kVStages;
                if (!mbar_wait(p_full, static_cast<uint32_t>(i) & 1u, abort) ||
                    !mbar_wait(&v_full[st], static_cast<uint32_t>(i / kVStages) & 1u, abort)) {
                    mok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t v_addr = smem_u32(sV + st * kTileBytes);
                const uint32_t p_tmem = tmem + kPCol + (i & 1) * (kKeys / 2);
#pragma unroll
                for (int kk = 0; kk < kKeys / 16; kk++)  // 16 keys = 8 columns of bf16 pairs
                    tc_mma_bf16_ts(tmem + kOCol, p_tmem + kk * 8, sdesc_sw128_mn(v_addr + kk * 2048, kHalf), idesc_pv,
                                   (i > 0 || kk > 0) ? 1u : 0u);
                tc_commit(&v_empty[st]);
                tc_commit(&pv_done[i & 1]);
            }
            if (!mok) {
                attn_timeout(a.status, abort);
                tc_commit(tdown);
                attn_drain(tdown, 0);
            }
        }
    } else {
        // ---------------------------------------------------------- softmax
        const uint32_t swz = static_cast<uint32_t>(r & 7);
        const int pair_bar = kPairBarrier0 + qd;
        if (nt > 0) {
            // RoPE of this thread's query row, in place: element t of the
            // first 64 and element t of the second 64 sit at the same
            // swizzled position of the two 16 KB halves; warpgroup wg
            // rotates chunks 4 wg .. 4 wg + 3
            if (!warp_wait(q_full, 0, abort)) {
                attn_timeout(a.status, abort);
                ok = false;
            }
            // rotated elements t (first half) and t + 64 (second half) of this
            // warpgroup's t in [32 wg, 32 wg + 32), as bf16 pairs for the TMEM
            // columns kQCol + t / 2 and kQCol + 32 + t / 2 (zeros past row B)
            uint32_t q1[16], q2[16];
            if (ok && b < a.B) {
                const float4* cs = reinterpret_cast<const float4*>(a.cs + (static_cast<size_t>(s) * a.B + b) * (kDh / 2));
#pragma unroll
                for (int cc = 0; cc < 4; cc++) {
                    const int c = wg * 4 + cc;
                    const uint8_t* p1 = sQ + r * 128 + ((static_cast<uint32_t>(c) ^ swz) << 4);
                    const uint4 x1 = *reinterpret_cast<const uint4*>(p1);
                    const uint4 x2 = *reinterpret_cast<const uint4*>(p1 + kHalf);
                    const uint32_t* u1 = reinterpret_cast<const uint32_t*>(&x1);
                    const uint32_t* u2 = reinterpret_cast<const uint32_t*>(&x2);
#pragma unroll
                    for (int e = 0; e < 4; e++) {
                        const float4 f = __ldg(cs + c * 4 + e);  // (cos, sin) of pairs 8c+2e, 8c+2e+1
                        const __nv_bfloat162 h1 = *reinterpret_cast<const __nv_bfloat162*>(&u1[e]);
                        const __nv_bfloat162 h2 = *reinterpret_cast<const __nv_bfloat162*>(&u2[e]);
                        const float a0 = __low2float(h1), a1 = __high2float(h1);
                        const float b0 = __low2float(h2), b1 = __high2float(h2);
                        q1[cc * 4 + e] = pack_bf16(a0 * f.x - b0 * f.y, a1 * f.z - b1 * f.w);
                        q2[cc * 4 + e] = pack_bf16(b0 * f.x + a0 * f.y, b1 * f.z + a1 * f.w);
                    }
                }
            } else {
#pragma unroll
                for (int k = 0; k < 16; k++) q1[k] = q2[k] = 0u;
            }
            tmem_st16u(tl + kQCol + wg * 16, q1);
            tmem_st16u(tl + kQCol + 32 + wg * 16, q2);
            tmem_wait_st();
            tc_fence_before();
            mbar_arrive(q_ready);
        }
        for (int i = 0; i < nt; i++) {
            const int j = j0 + i;
            // visible keys of this row among this warpgroup's 64 keys of the tile
            uint64_t w = 0ull;
            if (row_ok) {
                int kvalid;
                if (j < a.nct) {
                    kvalid = min(kKeys, a.C - j * kKeys);
                    w = ~0ull;
                } else {
                    const int t = j - a.nct;
                    kvalid = min(kKeys, nn - t * kKeys);
                    w = 2 * t + wg < a.mw ? __ldg(a.mask + (static_cast<size_t>(s) * a.B + b) * a.mw + 2 * t + wg) : 0ull;
                }
                kvalid -= cb;
                if (kvalid <= 0)
                    w = 0ull;
                else if (kvalid < 64)
                    w &= (1ull << kvalid) - 1ull;
            }
            const bool full = __all_sync(0xFFFFFFFFu, w == ~0ull);  // whole warp sees all 64 keys
            // Both warps of the lane quarter reach both pair barriers of every
            // iteration and leave the loop at the same point: a failed wait is
            // exchanged with the row max and acted on after the barriers.
            if (ok && !warp_wait(s_full, static_cast<uint32_t>(i) & 1u, abort)) {
                attn_timeout(a.status, abort);
                ok = false;
            }
            float sv[64];
            float mx = -INFINITY;
            if (ok) {
                tc_fence_after();
                tmem_ld64(tl + kSCol + cb, sv);
                // S is in registers: the buffer is free for S(i + 2)
                tc_fence_before();
                mbar_arrive(s_empty);
                if (full) {
#pragma unroll
                    for (int c = 0; c < 64; c += 2) mx = fmaxf(mx, fmaxf(sv[c], sv[c + 1]));
                } else {
#pragma unroll
                    for (int c = 0; c < 64; c++) {
                        if (!((w >> c) & 1ull)) sv[c] = -INFINITY;
                        mx = fmaxf(mx, sv[c]);
                    }
                }
            }
            xch[wg * kRows + r] = mx;
            if (lane == 0) xok[wg * 4 + qd] = ok ? 1 : 0;
            named_bar_sync(pair_bar, 64);
            mx = fmaxf(mx, xch[(1 - wg) * kRows + r]);
            ok = ok && xok[(1 - wg) * 4 + qd] != 0;
            named_bar_sync(pair_bar, 64);  // both read before the next tile's write
            if (!ok) break;
            const float mx2 = mx * a.sl2;
            const bool resc = mx2 > m_run + kRescaleSlack;
            const float m_new = resc ? mx2 : m_run;
            const float alpha = resc ? ex2(m_run - m_new) : 1.0f;
            // P buffer i & 1 was last read by PV(i - 2); O must be stable (PV(i - 1)
            // done) only when it is rescaled.  On a timeout this tile is
            // skipped; the pair leaves the loop together at the next exchange.
            if (i > 1 && !warp_wait(&pv_done[i & 1], (static_cast<uint32_t>(i >> 1) & 1u) ^ 1u, abort)) {
                attn_timeout(a.status, abort);
                ok = false;
                continue;
            }
            tc_fence_after();
            const bool any_resc = __any_sync(0xFFFFFFFFu, resc);
            if (i > 0 && any_resc) {
                if (!warp_wait(&pv_done[(i - 1) & 1], static_cast<uint32_t>((i - 1) >> 1) & 1u, abort)) {
                    attn_timeout(a.status, abort);
                    ok = false;
                    continue;
                }
                tc_fence_after();
                {
#pragma unroll
                    for (int c0 = 0; c0 < 64; c0 += 16) {
                        float o[16];
                        tmem_ld16(tl + kOCol + cb + c0, o);
#pragma unroll
                        for (int e = 0; e < 16; e++) o[e] *= alpha;
                        tmem_st16(tl + kOCol + cb + c0, o);
                    }
                    tmem_wait_st();
                }
            }
            l *= alpha;
            m_run = m_new;
            // P = 2^(s * scale * log2 e - m) as bf16 pairs into TMEM P buffer
            // i & 1 (lane = row, keys 64 wg .. 64 wg + 63 in 32 columns); masked
            // keys hold -inf and give 0 (so does every key of a row that has
            // seen no visible key: m = -inf)
            const float nm = m_run == -INFINITY ? 0.0f : -m_run;
            float lsum = 0.0f;
            uint32_t pk[32];
#pragma unroll
            for (int c = 0; c < 64; c += 2) {
                const float p0 = ex2(fmaf(sv[c], a.sl2, nm));
                const float p1 = ex2(fmaf(sv[c + 1], a.sl2, nm));
                lsum += p0 + p1;
                pk[c >> 1] = pack_bf16(p0, p1);
            }
            tmem_st32(tl + kPCol + (i & 1) * (kKeys / 2) + wg * 32, pk);
            tmem_wait_st();
            l += lsum;
            tc_fence_before();
            mbar_arrive(p_full);
        }
        if (ok && nt > 0) {
            if (!warp_wait(&pv_done[(nt - 1) & 1], static_cast<uint32_t>((nt - 1) >> 1) & 1u, abort)) {
                attn_timeout(a.status, abort);
                ok = false;
            }
            tc_fence_after();
        }
        // the row sum is split over the two warpgroups
        xch[wg * kRows + r] = l;
        named_bar_sync(pair_bar, 64);
        l += xch[(1 - wg) * kRows + r];
        ok = __all_sync(0xFFFFFFFFu, ok);
    }

    const int h = kvh * a.G + g;
    if (a.splits == 1) {
        if (warp >= 2 && ok) {
            float* orow = a.out + ((static_cast<size_t>(s) * a.B + b) * a.Hq + h) * kDh + cb;
            const float inv = (row_ok && l > 0.0f) ? 1.0f / l : 0.0f;
#pragma unroll
            for (int c0 = 0; c0 < 64; c0 += 16) {
                float o[16];
                if (nt > 0) {
                    tmem_ld16(tl + kOCol + cb + c0, o);
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
        // Split key range.  Columns are owned in groups of 4: CTA j merges
        // [c_lo(j), c_hi(j)).  After a cluster barrier (every CTA is past its
        // main loop, so the K and V rings are free), every CTA p pushes,
        // with 16-byte stores into the peers' shared memory, its (m, l) row
        // to every peer and its unnormalised O row slices to their owners
        // (row-major, row stride padded to an odd number of 16-byte units:
        // conflict-free); after a second barrier CTA j merges locally, in
        // rank order: O = sum_p 2^(m_p - M) O_p / sum_p 2^(m_p - M) l_p.
        float* rbuf = reinterpret_cast<float*>(sK);     // [p][128 rows][stride]
        float2* rml = reinterpret_cast<float2*>(sV);    // [p][128 rows]
        __syncwarp();
        cluster_sync_all();
        if (warp >= 2) {
            const bool have = ok && nt > 0;
            if (wg == 0)
                for (int jj = 0; jj < a.splits; jj++)
                    st_cluster_f32x2(smem_u32(rml + split * kRows + r), jj, m_run, have ? l : 0.0f);
            if (have) {
                float o[64];
                tmem_ld64(tl + kOCol + cb, o);
                for (int jj = 0; jj < a.splits; jj++) {
                    const int lo = slice_lo(jj, a.splits), ncol = slice_lo(jj + 1, a.splits) - lo;
                    const int stride = slice_stride(ncol);
                    const uint32_t dst = smem_u32(rbuf + (split * kRows + r) * stride);
#pragma unroll
                    for (int c = 0; c < 64; c += 4)
                        if (cb + c >= lo && cb + c < lo + ncol)
                            st_cluster_f32x4(dst + (cb + c - lo) * 4, jj, o[c], o[c + 1], o[c + 2], o[c + 3]);
                }
            }
        }
        __syncwarp();
        cluster_sync_all();  // every push has landed
        if (warp >= 2) {
            const int c_lo = slice_lo(split, a.splits), ncol = slice_lo(split + 1, a.splits) - c_lo;
            const int stride = slice_stride(ncol);
            float M = -INFINITY;
            for (int p = 0; p < a.splits; p++) {
                const float2 ml = rml[p * kRows + r];
                if (ml.y > 0.0f) M = fmaxf(M, ml.x);
            }
            float wp[kMaxSplits];
            float L = 0.0f;
#pragma unroll
            for (int p = 0; p < kMaxSplits; p++) {
                wp[p] = 0.0f;
                if (p < a.splits) {
                    const float2 ml = rml[p * kRows + r];
                    if (ml.y > 0.0f) {
                        wp[p] = ex2(ml.x - M);
                        L += wp[p] * ml.y;
                    }
                }
            }
            const float inv = (row_ok && L > 0.0f) ? 1.0f / L : 0.0f;
            if (b < a.B) {
                float* orow = a.out + ((static_cast<size_t>(s) * a.B + b) * a.Hq + h) * kDh + c_lo;
                // the two warpgroups take alternate 4-column groups of the slice
                for (int c = 4 * wg; c < ncol; c += 8) {
                    float4 o = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
#pragma unroll
                    for (int p = 0; p < kMaxSplits; p++) {
                        if (wp[p] != 0.0f) {
                            const float4 v = *reinterpret_cast<const float4*>(rbuf + (p * kRows + r) * stride + c);
                            o.x += wp[p] * v.x;
                            o.y += wp[p] * v.y;
                            o.z += wp[p] * v.z;
                            o.w += wp[p] * v.w;
                        }
                    }
                    *reinterpret_cast<float4*>(orow + c) = make_float4(o.x * inv, o.y * inv, o.z * inv, o.w * inv);
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
};

// Workspace: rotated tree keys, then the (cos, sin) table (no device query).
struct WsLayout {
    size_t off_kr, off_cs, total;
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
    if (static_cast<long long>(c->nseq) * c->B * (c->Hq + c->Hkv) > (1ll << 30)) return false;
    if (static_cast<long long>(c->C) * c->Hkv * kDh > (1ll << 40)) return false;
    return true;
}

// Splits of the key list (= cluster size): as many as keep every CTA in one
// wave (1 CTA per SM) with at least two key tiles per split.
int pick_splits(int blocks, int max_tiles, int nsm) {
    int sp = 1;
    while (sp < kMaxSplits && static_cast<long long>(blocks) * (sp + 1) <= nsm && max_tiles / (sp + 1) >= 2) sp++;
    return sp;
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
    return p;
}

WsLayout ws_layout(const dart_attn_config* c) {
    WsLayout w;
    const size_t kr = static_cast<size_t>(c->nseq) * c->B * c->Hkv * kDh * 2;
    const size_t cs = static_cast<size_t>(c->nseq) * c->B * (kDh / 2) * 8;
    w.off_kr = 0;
    w.off_cs = align256(w.off_kr + kr);
    w.total = align256(w.off_cs + cs);
    return w;
}

// Compute capability, shared-memory opt-in and SM count of a device, queried
// once per device.
struct DevInfo {
    int major, minor, optin, nsm;
};
bool dev_info(int dev, DevInfo* out) {
    constexpr int kMaxDev = 64;
    static DevInfo info[kMaxDev];
    static std::atomic<int> ready[kMaxDev];
    if (dev < 0 || dev >= kMaxDev) return false;
    if (ready[dev].load(std::memory_order_acquire) == 0) {
        DevInfo d{};
        if (cudaDeviceGetAttribute(&d.major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&d.minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&d.optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&d.nsm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
            return false;
        info[dev] = d;  // every thread that gets here writes the same values
        ready[dev].store(1, std::memory_order_release);
    }
    *out = info[dev];
    return true;
}

// Queries [nseq][B][Hq][dh] bf16 with a (64, G heads, qpt rows, 1) box: the
// 128 box rows are (tree row, head) pairs, heads fastest.
bool encode_q(CUtensorMap* m, const void* base, int nseq, int B, int Hq, int G, int qpt) {
    EncodeTiledFn fn = tensor_map_encoder();
    if (!fn) return false;
    cuuint64_t dims[4] = {static_cast<cuuint64_t>(kDh), static_cast<cuuint64_t>(Hq), static_cast<cuuint64_t>(B),
                          static_cast<cuuint64_t>(nseq)};
    cuuint64_t strides[3] = {static_cast<cuuint64_t>(kDh) * 2, static_cast<cuuint64_t>(Hq) * kDh * 2,
                             static_cast<cuuint64_t>(B) * Hq * kDh * 2};
    cuuint32_t box[4] = {64, static_cast<cuuint32_t>(G), static_cast<cuuint32_t>(qpt), 1};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, estr,
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

// The kernel's shared-memory opt-in, set once per device (a host call that
// costs microseconds when repeated on every launch).
bool attn_attr_set(int dev) {
    static std::atomic<uint64_t> done{0};
    const uint64_t bit = dev < 64 ? (1ull << dev) : 0ull;
    if (bit && (done.load() & bit)) return true;
    if (cudaFuncSetAttribute(tree_attn_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kAttnSmem) !=
        cudaSuccess)
        return false;
    done.fetch_or(bit);
    return true;
}



// Validates, then enqueues the pre-pass and the attention kernel; ev[0..2]
// (optional) are recorded before the pre-pass, between the two and after.
int enqueue_tree_attention(const dart_attn_config* cfg, const void* q, const void* k_tree, const void* v_tree,
                           const void* k_ctx, const void* v_ctx, const int32_t* pos_ids, const uint64_t* mask,
                           const int32_t* n_nodes, float* out, void* workspace, size_t workspace_bytes,
                           int* status, void* stream, cudaEvent_t* ev) {
    if (!valid_cfg(cfg)) return DART_ERR_INVALID;
    const dart_attn_config& c = *cfg;
    if (!q || !k_tree || !v_tree || !pos_ids || !mask || !n_nodes || !out || !workspace) return DART_ERR_INVALID;
    if (c.C > 0 && (!k_ctx || !v_ctx)) return DART_ERR_INVALID;
    if (!al16(q) || !al16(k_tree) || !al16(v_tree) || !al16(out) || !al16(mask) || !al16(pos_ids) ||
        !al16(n_nodes) || (reinterpret_cast<uintptr_t>(workspace) & 255u))
        return DART_ERR_INVALID;
    if (c.C > 0 && (!al16(k_ctx) || !al16(v_ctx))) return DART_ERR_INVALID;
    if (status && !al16(status)) return DART_ERR_INVALID;
    const WsLayout wl = ws_layout(cfg);
    if (workspace_bytes < wl.total) return DART_ERR_INVALID;
    int dev = 0;
    DevInfo di;
    if (cudaGetDevice(&dev) != cudaSuccess || !dev_info(dev, &di)) return DART_ERR_CUDA;
    if (di.major != 10 || di.minor != 3 || di.optin < kAttnSmem) return DART_ERR_UNSUPPORTED;
    const int nsm = di.nsm > 0 ? di.nsm : 148;
    const Plan p = make_plan(cfg, nsm);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    uint8_t* ws = static_cast<uint8_t*>(workspace);
    __nv_bfloat16* kr = reinterpret_cast<__nv_bfloat16*>(ws + wl.off_kr);
    float2* cs = reinterpret_cast<float2*>(ws + wl.off_cs);

    CUtensorMap tmQ, tmKc, tmVc, tmKt, tmVt;
    if (!encode_q(&tmQ, q, c.nseq, c.B, c.Hq, p.G, p.qpt)) return DART_ERR_CUDA;
    if (!encode_kv(&tmKt, kr, c.nseq, c.B, c.Hkv) || !encode_kv(&tmVt, v_tree, c.nseq, c.B, c.Hkv))
        return DART_ERR_CUDA;
    if (c.C > 0) {
        if (!encode_kv(&tmKc, k_ctx, c.nseq, c.C, c.Hkv) || !encode_kv(&tmVc, v_ctx, c.nseq, c.C, c.Hkv))
            return DART_ERR_CUDA;
    } else {
        tmKc = tmKt;  // never read: no context tiles
        tmVc = tmVt;
    }

    PrepArgs ra;
    std::memset(&ra, 0, sizeof ra);
    ra.nseq = c.nseq;
    ra.B = c.B;
    ra.Hkv = c.Hkv;
    ra.kt = static_cast<const __nv_bfloat16*>(k_tree);
    ra.pos_ids = pos_ids;
    ra.kr = kr;
    ra.cs = cs;
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
    aa.cs = cs;
    aa.n_nodes = n_nodes;
    aa.mask = mask;
    aa.out = out;
    aa.status = status;

    if (!attn_attr_set(dev)) return DART_ERR_CUDA;
    const int prep_blocks = static_cast<int>(std::min<long long>(
        (static_cast<long long>(c.nseq) * c.B * c.Hkv + 7) / 8, 16LL * nsm));  // 8 rows per block
    if (ev && cudaEventRecord(ev[0], st) != cudaSuccess) return DART_ERR_CUDA;
    if (launch_pdl(attn_prep_kernel, dim3(prep_blocks), dim3(256), 0, st, ra) != cudaSuccess) return DART_ERR_CUDA;
    if (ev && cudaEventRecord(ev[1], st) != cudaSuccess) return DART_ERR_CUDA;
    const cudaError_t le =
        p.splits > 1 ? launch_pdl_cluster(tree_attn_kernel, dim3(p.blocks * p.splits), dim3(kAttnThreads), kAttnSmem,
                                          st, p.splits, tmQ, tmKc, tmVc, tmKt, tmVt, aa)
                     : launch_pdl(tree_attn_kernel, dim3(p.blocks), dim3(kAttnThreads), kAttnSmem, st, tmQ, tmKc,
                                  tmVc, tmKt, tmVt, aa);
    if (le != cudaSuccess) return DART_ERR_CUDA;
    if (ev && cudaEventRecord(ev[2], st) != cudaSuccess) return DART_ERR_CUDA;
    return DART_OK;
}

}  // namespace
}  // namespace dart

using namespace dart;

extern "C" {

size_t dart_tree_attention_workspace(const dart_attn_config* cfg) {
    if (!valid_cfg(cfg)) return 0;
    return ws_layout(cfg).total;
}


int dart_tree_attention(const dart_attn_config* cfg, const void* q, const void* k_tree, const void* v_tree,
                        const void* k_ctx, const void* v_ctx, const int32_t* pos_ids, const uint64_t* mask,
                        const int32_t* n_nodes, float* out, void* workspace, size_t workspace_bytes, int* status,
                        void* stream) {
    return enqueue_tree_attention(cfg, q, k_tree, v_tree, k_ctx, v_ctx, pos_ids, mask, n_nodes, out, workspace,
                                  workspace_bytes, status, stream, nullptr);
}

int dart_tree_attention_timed(const dart_attn_config* cfg, const void* q, const void* k_tree, const void* v_tree,
                              const void* k_ctx, const void* v_ctx, const int32_t* pos_ids, const uint64_t* mask,
                              const int32_t* n_nodes, float* out, void* workspace, size_t workspace_bytes,
                              int* status, float* ms_rope, float* ms_attn, void* stream) {
    if (!ms_rope || !ms_attn) return DART_ERR_INVALID;
    cudaEvent_t ev[3] = {nullptr, nullptr, nullptr};
    int rc = DART_OK;
    for (int i = 0; i < 3 && rc == DART_OK; i++)
        if (cudaEventCreate(&ev[i]) != cudaSuccess) rc = DART_ERR_CUDA;
    if (rc == DART_OK)
        rc = enqueue_tree_attention(cfg, q, k_tree, v_tree, k_ctx, v_ctx, pos_ids, mask, n_nodes, out, workspace,
                                    workspace_bytes, status, stream, ev);
    if (rc == DART_OK && cudaEventSynchronize(ev[2]) != cudaSuccess) rc = DART_ERR_CUDA;
    if (rc == DART_OK && (cudaEventElapsedTime(ms_rope, ev[0], ev[1]) != cudaSuccess ||
                          cudaEventElapsedTime(ms_attn, ev[1], ev[2]) != cudaSuccess))
        rc = DART_ERR_CUDA;
    for (int i = 0; i < 3; i++)
        if (ev[i]) cudaEventDestroy(ev[i]);
    return rc;
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
