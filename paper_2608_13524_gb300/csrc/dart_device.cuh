// Device-side building blocks of the DARTree construction path (sm_103a):
// inline-PTX wrappers for mbarrier / TMA / tcgen05, order-preserving 64-bit
// selection keys, a block-wide radix select, and the fused LM-head epilogue
// (online log-sum-exp + per-node top-k) shared by the bf16 tensor-core kernel
// and the fp32 CUDA-core kernel.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace dart {

// Device status word bits (read back by dart_status_sync).
constexpr int kDevTimeout = 1;      // a bounded wait gave up
constexpr int kDevOrphan = 2;       // pruning kept a node whose parent was cut (impossible for beta <= 0)
constexpr int kDevBounds = 4;       // debug builds: a data-dependent index failed its check

// Debug builds (-DDART_DEBUG) check data-dependent indices (parent slots,
// token ids, output positions) before they are used: a failed check sets
// kDevBounds in the status word and the caller skips the access, so the
// context stays usable and dart_status_sync reports DART_ERR_BOUNDS.
// Release builds compile the checks away (the function returns true).
__device__ __forceinline__ bool bounds_check(int* status, bool ok) {
#ifdef DART_DEBUG
    if (!ok && status) atomicOr(status, kDevBounds);
    return ok;
#else
    (void)status;
    (void)ok;
    return true;
#endif
}

// A wait that has not completed after this long means a bug; give up.
constexpr unsigned long long kWaitLimitNs = 2000000000ull;  // 2 s

constexpr int kNPadMax = 256;       // max nodes per depth (nseq * W)
constexpr int kTileM = 128;         // MMA M: vocabulary rows / output features per tile
constexpr int kBlockK = 64;         // bf16 elements per 128-byte swizzled row
constexpr int kCandCap = 128;       // per-node candidate slots per tile (one tile worth)
constexpr int kCandCapLarge = 32;   // slots per node for 128-node groups (overflow: more merge rounds)
constexpr int kEpiBarrier = 1;      // named barrier id used by the epilogue warps

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// x = hi + lo with hi = bf16(x) and lo = bf16(x - hi): ~16 mantissa bits of
// x as two tensor-core operands.
__device__ __forceinline__ void split_bf16(float x, __nv_bfloat16& hi, __nv_bfloat16& lo) {
    hi = __float2bfloat16_rn(x);
    lo = __float2bfloat16_rn(x - __bfloat162float(hi));
}

// Thread-block clusters: rank in the cluster, a barrier over every thread of
// every CTA of the cluster (release / acquire: shared-memory writes before it
// are visible to the whole cluster after it), and a 4-byte load from the
// shared memory of CTA `rank` at the offset of the local address `local`.
__device__ __forceinline__ uint32_t cluster_ctarank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
__device__ __forceinline__ void cluster_sync_all() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ float ld_cluster_f32(uint32_t local, uint32_t rank) {
    uint32_t remote;
    float v;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(local), "r"(rank));
    asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(remote) : "memory");
    return v;
}

__device__ __forceinline__ unsigned long long globaltimer_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Programmatic dependent launch.  pdl_trigger lets the next kernel of the
// stream start its prologue early; pdl_wait blocks until every prerequisite
// kernel has completed and its memory is visible.  Every kernel calls
// pdl_wait before it touches data written by an earlier kernel (or data an
// earlier kernel still reads), so completion is transitive along the stream.
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

__device__ __forceinline__ void named_bar_sync(int id, int nthreads) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

// ------------------------------------------------------------------ mbarrier

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
        " selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}
// Waits for the phase with the given parity.  Gives up (returns false) when
// *abort becomes nonzero or after limit_ns (kWaitLimitNs unless a test asks
// for a shorter limit).
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, volatile int* abort,
                                          unsigned long long limit_ns = kWaitLimitNs) {
    if (mbar_try_wait(bar, parity)) return true;
    const unsigned long long t0 = globaltimer_ns();
    for (;;) {
        if (mbar_try_wait(bar, parity)) return true;
        if (*abort) return false;
        if (globaltimer_ns() - t0 > limit_ns) return false;
    }
}

// ----------------------------------------------------------------------- TMA

__device__ __forceinline__ uint64_t l2_policy_evict_first() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    return p;
}
__device__ __forceinline__ uint64_t l2_policy_evict_last() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
    return p;
}
// 2-D tiled bulk copy global -> shared, completing on `bar` (x = innermost).
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, uint64_t* bar, int x, int y,
                                            uint64_t policy) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%0], [%1, {%3, %4}], [%2], %5;" ::"r"(smem_u32(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(x), "r"(y), "l"(policy)
        : "memory");
}

// One bulk copy global -> shared (both 16-byte aligned, bytes a multiple of
// 16), completing on `bar`.
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                     smem_u32(dst)),
                 "l"(src), "r"(bytes), "r"(smem_u32(bar))
                 : "memory");
}

// L2 prefetch of one tile of a 2-D tensor (no shared memory, no barrier).
__device__ __forceinline__ void tma_prefetch_2d(const CUtensorMap* map, int x, int y) {
    asm volatile("cp.async.bulk.prefetch.tensor.2d.L2.global.tile [%0, {%1, %2}];" ::"l"(reinterpret_cast<uint64_t>(map)),
                 "r"(x), "r"(y)
                 : "memory");
}

// ------------------------------------------------------------------- tcgen05

__device__ __forceinline__ void tmem_alloc(uint32_t* slot, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(slot)),
                 "r"(ncols)
                 : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// D[tmem] (+)= A[smem] * B[smem]^T, bf16 inputs, fp32 accumulation.
__device__ __forceinline__ void tc_mma_bf16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                            uint32_t accumulate) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
        " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(tmem_d),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}
// Arrives once on `bar` when every tcgen05 op issued so far by this thread is done.
__device__ __forceinline__ void tc_commit(uint64_t* bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                     smem_u32(bar))
                 : "memory");
}
// 32 TMEM lanes x 16 consecutive 32-bit columns: thread i of the warp gets lane
// (warp's lane quarter + i), columns [col, col+16).
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16]) {
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15},"
        " [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
    // the registers are tied to the wait so no use can move above it
    asm volatile("tcgen05.wait::ld.sync.aligned;"
                 : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]),
                   "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]),
                   "+r"(r[14]), "+r"(r[15])
                 :
                 : "memory");
#pragma unroll
    for (int i = 0; i < 16; i++) v[i] = __uint_as_float(r[i]);
}

// Two 32x32b.x16 loads (e.g. the hi and lo halves of an accumulator) with a
// single wait.
__device__ __forceinline__ void tmem_ld16_pair(uint32_t ta, uint32_t tb, float (&va)[16], float (&vb)[16]) {
    uint32_t r[16], q[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15},"
        " [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(ta));
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15},"
        " [%16];"
        : "=r"(q[0]), "=r"(q[1]), "=r"(q[2]), "=r"(q[3]), "=r"(q[4]), "=r"(q[5]), "=r"(q[6]), "=r"(q[7]),
          "=r"(q[8]), "=r"(q[9]), "=r"(q[10]), "=r"(q[11]), "=r"(q[12]), "=r"(q[13]), "=r"(q[14]), "=r"(q[15])
        : "r"(tb));
    asm volatile("tcgen05.wait::ld.sync.aligned;"
                 : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]),
                   "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]),
                   "+r"(r[14]), "+r"(r[15]), "+r"(q[0]), "+r"(q[1]), "+r"(q[2]), "+r"(q[3]), "+r"(q[4]),
                   "+r"(q[5]), "+r"(q[6]), "+r"(q[7]), "+r"(q[8]), "+r"(q[9]), "+r"(q[10]), "+r"(q[11]),
                   "+r"(q[12]), "+r"(q[13]), "+r"(q[14]), "+r"(q[15])
                 :
                 : "memory");
#pragma unroll
    for (int i = 0; i < 16; i++) {
        va[i] = __uint_as_float(r[i]);
        vb[i] = __uint_as_float(q[i]);
    }
}

// Shared-memory matrix descriptor of a K-major operand tile written by TMA
// with 128-byte swizzling: rows of 128 bytes, 8-row groups 1024 bytes apart
// (stride byte offset), tile base 1024-byte aligned; the leading byte offset
// is unused because one MMA's K extent (32 bytes) stays inside a swizzle row.
__device__ __forceinline__ uint64_t sdesc_sw128(uint32_t saddr) {
    uint64_t d = 0;
    d |= static_cast<uint64_t>((saddr >> 4) & 0x3FFFu);          // start address >> 4
    d |= static_cast<uint64_t>((1024u >> 4) & 0x3FFFu) << 32;    // stride byte offset >> 4
    d |= static_cast<uint64_t>(1u) << 46;                        // descriptor version (tcgen05)
    d |= static_cast<uint64_t>(2u) << 61;                        // swizzle mode: 128B
    return d;
}
// Instruction descriptor, kind::f16: D fp32, A and B bf16, both K-major.
__host__ __device__ constexpr uint32_t idesc_bf16_f32(int M, int N) {
    return (1u << 4) | (1u << 7) | (1u << 10) | (static_cast<uint32_t>(N >> 3) << 17) |
           (static_cast<uint32_t>(M >> 4) << 24);
}

// ---------------------------------------------------------------- selection
//
// A candidate is a 64-bit key whose unsigned order is the selection order:
// high word = order-preserving image of the fp32 value (larger value =
// larger key), low word = ~index (smaller index wins ties).  Key 0 is below
// every real candidate and marks empty slots.

__device__ __forceinline__ uint32_t f32_ord(float f) {
    uint32_t u = __float_as_uint(f);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float f32_unord(uint32_t o) {
    uint32_t u = (o & 0x80000000u) ? (o & 0x7FFFFFFFu) : ~o;
    return __uint_as_float(u);
}
__device__ __forceinline__ uint64_t make_key(float v, uint32_t idx) {
    if (v == 0.0f) v = 0.0f;  // -0 and +0 compare equal
    return (static_cast<uint64_t>(f32_ord(v)) << 32) | static_cast<uint64_t>(0xFFFFFFFFu - idx);
}
__device__ __forceinline__ float key_val(uint64_t key) { return f32_unord(static_cast<uint32_t>(key >> 32)); }
__device__ __forceinline__ uint32_t key_idx(uint64_t key) {
    return 0xFFFFFFFFu - static_cast<uint32_t>(key & 0xFFFFFFFFull);
}

// Block-wide radix select: returns the kk-th largest of the n keys in shared
// memory (1 <= kk <= n; keys distinct except for zeros).  Uses `hist` (256
// u32) and `scal` (2 ints) of shared scratch.  Every thread of the block must
// call it; it synchronises the block.
__device__ __forceinline__ uint64_t block_kth_largest(const uint64_t* keys, int n, int kk, uint32_t* hist,
                                                      int* scal) {
    uint64_t prefix = 0, mask = 0;
    int remaining = kk;
    const int tid = threadIdx.x, nt = blockDim.x;
    for (int shift = 56; shift >= 0; shift -= 8) {
        for (int i = tid; i < 256; i += nt) hist[i] = 0;
        __syncthreads();
        for (int i = tid; i < n; i += nt) {
            const uint64_t e = keys[i];
            if ((e & mask) == prefix) atomicAdd(&hist[(e >> shift) & 255u], 1u);
        }
        __syncthreads();
        if (tid < 32) {
            // lane l owns digits 255-8l .. 248-8l (highest digits first)
            uint32_t loc[8];
            uint32_t sum = 0;
#pragma unroll
            for (int j = 0; j < 8; j++) {
                loc[j] = hist[255 - 8 * tid - j];
                sum += loc[j];
            }
            uint32_t incl = sum;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                uint32_t t = __shfl_up_sync(0xFFFFFFFFu, incl, o);
                if (tid >= o) incl += t;
            }
            const unsigned hit = __ballot_sync(0xFFFFFFFFu, incl >= static_cast<uint32_t>(remaining));
            const int lane = __ffs(hit) - 1;
            if (tid == lane) {
                uint32_t cum = incl - sum;
                int digit = 255 - 8 * lane;
#pragma unroll
                for (int j = 0; j < 8; j++) {
                    if (cum + loc[j] >= static_cast<uint32_t>(remaining)) {
                        digit = 255 - 8 * lane - j;
                        break;
                    }
                    cum += loc[j];
                }
                scal[0] = digit;
                scal[1] = remaining - static_cast<int>(cum);
            }
        }
        __syncthreads();
        prefix |= static_cast<uint64_t>(scal[0]) << shift;
        mask |= 255ull << shift;
        remaining = scal[1];
        __syncthreads();
    }
    return prefix;
}

constexpr int kRankMax = 1024;  // candidate count up to which an O(n^2 / threads) rank sort is used

// Writes the kk largest nonzero keys, in descending order, to out[0..kk).
// `keys` holds nlists lists of `len` keys, each sorted in descending order
// with zeros (empty slots) last; at least kk keys are nonzero.  Only keys
// >= a threshold T can be among the kk largest, where T is the larger of
// `bound` (0, or a key known to have kk keys >= it, such as the largest
// k-th key any LM-head CTA published for the node) and the kk-th largest
// list head (some kk lists reach it; skipped when rank_heads is false); the
// survivors are ranked by counting.
// A block-wide radix select handles a survivor set larger than kRankMax.
// `surv` has kRankMax slots.  Every thread of the block must call this.
__device__ __forceinline__ void topk_of_sorted_lists(const uint64_t* keys, int nlists, int len, int kk,
                                                     uint64_t bound, uint64_t* out, uint64_t* surv, uint64_t* thr,
                                                     uint32_t* hist, int* scal, bool rank_heads = true) {
    const int tid = threadIdx.x, nt = blockDim.x;
    const int n = nlists * len;
    if (tid == 0) {
        *thr = 0ull;
        scal[2] = 0;
    }
    __syncthreads();
    if (rank_heads && nlists >= kk && nlists > 1) {
        for (int r = tid; r < nlists; r += nt) {
            const uint64_t h = keys[r * len];
            if (h == 0ull) continue;
            int rank = 0;
            int q = 0;
            for (; q + 8 <= nlists; q += 8) {
#pragma unroll
                for (int u = 0; u < 8; u++) rank += keys[(q + u) * len] > h;
            }
            for (; q < nlists; q++) rank += keys[q * len] > h;
            if (rank == kk - 1) *thr = h;
        }
        __syncthreads();
    }
    const uint64_t T = *thr > bound ? *thr : bound;
    for (int i = tid; i < n; i += nt) {
        const uint64_t x = keys[i];
        if (x != 0ull && x >= T) {
            const int pos = atomicAdd(&scal[2], 1);
            if (pos < kRankMax) surv[pos] = x;
        }
    }
    __syncthreads();
    const int m = scal[2];
    if (m > kRankMax) {
        const uint64_t kth = block_kth_largest(keys, n, kk, hist, scal);
        if (tid == 0) scal[2] = 0;
        __syncthreads();
        for (int i = tid; i < n; i += nt) {
            const uint64_t x = keys[i];
            if (x != 0ull && x >= kth) surv[atomicAdd(&scal[2], 1)] = x;
        }
        __syncthreads();
    }
    const int mm = m > kRankMax ? kk : m;
    for (int i = tid; i < mm; i += nt) {
        const uint64_t x = surv[i];
        int r = 0;
        int j = 0;
        for (; j + 8 <= mm; j += 8) {
#pragma unroll
            for (int u = 0; u < 8; u++) r += surv[j + u] > x;
        }
        for (; j < mm; j++) r += surv[j] > x;
        if (r < kk) out[r] = x;
    }
    __syncthreads();
}

// Block-wide sums (every thread gets the total; `red` holds one value per warp).
__device__ __forceinline__ int block_sum_int(int v, int* red) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
    __syncthreads();
    if (lane == 0) red[warp] = v;
    __syncthreads();
    int t = 0;
    for (int i = 0; i < nw; i++) t += red[i];
    return t;
}

__device__ __forceinline__ float block_sum_float(float v, float* red) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
    __syncthreads();
    if (lane == 0) red[warp] = v;
    __syncthreads();
    float t = 0.0f;
    for (int i = 0; i < nw; i++) t += red[i];
    return t;
}

// ------------------------------------------------ fused LM-head epilogue
//
// Every epilogue thread owns one vocabulary row of a 128-row tile and sees
// the scaled logits of its row for the CTA's node group, 16 nodes (one
// "chunk") at a time.  Per node it keeps:
//   * log-sum-exp: per warp, a reference max m_ref (shared memory) and a
//     running sum of exp(z - m_ref) (a register of the lanes 2j, 2j+1 after
//     the butterfly reduction).  m_ref is raised -- and the sum rescaled --
//     only when some logit exceeds it by more than kRefSlack, so after the
//     first tile the exact warp max is almost never needed;
//   * top-k: a CTA-wide list of keys (shared memory, sorted).  A logit
//     enters the tile's candidate buffer only if it beats the node's current
//     k-th key; after the tile one warp per node merges the candidates.

constexpr unsigned kFull = 0xFFFFFFFFu;
constexpr float kRefSlack = 30.0f;  // exp(30) ~ 1e13: sums stay far from fp32 overflow

struct EpiSmem {
    uint64_t* list;   // [NG][k]   sorted desc, 0 = empty
    uint64_t* cand;   // [NG][cap]
    uint64_t* gcache; // [NG]  filter threshold: max(own k-th key, last seen cross-CTA bound) (see epi_merge)
    int* cnt;         // [NG]  candidates offered this round (may exceed cap)
    int* more;        // [2]   "a candidate found no free slot" flags of alternate merge rounds
    float* mref;      // [4][NG]  per-warp reference max
    float2* stats;    // [4][NG]  (reference, sum exp) per epilogue warp at the end
    int cap;          // candidate slots per node
};

// (m, s) <- (m, s) (+) (m2, s2) for sums of exp relative to their maxima.
__device__ __forceinline__ float2 lse_merge(float2 a, float2 b) {
    if (b.x == -INFINITY) return a;
    if (a.x == -INFINITY) return b;
    const float m = fmaxf(a.x, b.x);
    return make_float2(m, a.y * __expf(a.x - m) + b.y * __expf(b.x - m));
}

// Reduce-scatter of 32 partial sums per lane across the warp: afterwards
// lane l holds, in v[0], the sum over the 32 lanes of v[l] (fixed order:
// 31 shuffles for 32 results).
__device__ __forceinline__ void warp_reduce_scatter32(float (&v)[32], int lane) {
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) {
        const bool up = (lane & o) != 0;
#pragma unroll
        for (int j = 0; j < o; j++) {
            const float send = up ? v[j] : v[j + o];
            const float recv = __shfl_xor_sync(kFull, send, o);
            v[j] = (up ? v[j + o] : v[j]) + recv;
        }
    }
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(kFull, v, o));
    return v;
}

// Butterfly reduction of 16 values per lane over the warp: returns, in
// lanes 2j and 2j+1, the reduction of v[j] over all 32 lanes (16 shuffles).
template <bool kMax>
__device__ __forceinline__ float bfly16(const float (&v)[16], int lane) {
    auto op = [](float x, float y) { return kMax ? fmaxf(x, y) : x + y; };
    float a[8], b[4], c[2];
    const bool h4 = lane & 16, h3 = lane & 8, h2 = lane & 4, h1 = lane & 2;
#pragma unroll
    for (int i = 0; i < 8; i++) a[i] = op(h4 ? v[8 + i] : v[i], __shfl_xor_sync(kFull, h4 ? v[i] : v[8 + i], 16));
#pragma unroll
    for (int i = 0; i < 4; i++) b[i] = op(h3 ? a[4 + i] : a[i], __shfl_xor_sync(kFull, h3 ? a[i] : a[4 + i], 8));
#pragma unroll
    for (int i = 0; i < 2; i++) c[i] = op(h2 ? b[2 + i] : b[i], __shfl_xor_sync(kFull, h2 ? b[i] : b[2 + i], 4));
    const float d = op(h1 ? c[1] : c[0], __shfl_xor_sync(kFull, h1 ? c[0] : c[1], 2));
    return op(d, __shfl_xor_sync(kFull, d, 1));
}

// The kk-th largest (1 <= kk <= R) of the R values y[0..R) (R a multiple of
// 32, at most 256), by one warp: MSB-first radix select over the values'
// order-preserving images; NaN if some value is NaN.
__device__ __forceinline__ float warp_kth_largest(const float* y, int R, int kk, int lane) {
    uint32_t u[8];
    bool nan = false;
#pragma unroll
    for (int q = 0; q < 8; q++) {
        const float v = q * 32 < R ? __ldcg(y + q * 32 + lane) : -INFINITY;
        nan |= isnan(v);
        u[q] = f32_ord(v);
    }
    if (__any_sync(kFull, nan)) return __int_as_float(0x7FC00000);
    uint32_t prefix = 0, mask = 0;
    int need = kk;
    for (int b = 31; b >= 0; b--) {
        const uint32_t bit = 1u << b, cand = prefix | bit, m2 = mask | bit;
        int cnt = 0;
#pragma unroll
        for (int q = 0; q < 8; q++)
            if (q * 32 < R) cnt += __popc(__ballot_sync(kFull, (u[q] & m2) == cand));
        if (cnt >= need)
            prefix = cand;
        else
            need -= cnt;
        mask = m2;
    }
    return f32_unord(prefix);
}

// nthr = number of epilogue threads (4 warps per 16-node chunk of the group).
// The first tile's filter starts from the node's published bound gthr[n0+i]
// (zero before the first merge), raised with seed scores (seed_y[n][0..R),
// launch_seed_score) to their k-th largest, which the CTAs of the first
// vocabulary range publish into gthr.  Called after the wait on the
// previous kernel.
__device__ __forceinline__ void epi_init(const EpiSmem& e, int NG, int k, int etid, int nthr,
                                         uint64_t* gthr = nullptr, int n0 = 0, int N = 0,
                                         const float* seed_y = nullptr, int seed_R = 0, bool publish = false) {
    for (int i = etid; i < NG * k; i += nthr) e.list[i] = 0ull;
    for (int i = etid; i < NG; i += nthr) {
        e.cnt[i] = 0;
        if (!seed_y)
            e.gcache[i] = (gthr && n0 + i < N) ? __ldcg(reinterpret_cast<const unsigned long long*>(gthr) + n0 + i) : 0ull;
    }
    if (seed_y) {
        const int lane = etid & 31;
        for (int i = etid >> 5; i < NG; i += nthr >> 5) {
            uint64_t g = 0ull;
            if (n0 + i < N) {
                const float b = warp_kth_largest(seed_y + static_cast<size_t>(n0 + i) * seed_R, seed_R, k, lane);
                if (gthr) g = __ldcg(reinterpret_cast<const unsigned long long*>(gthr) + n0 + i);
                if (isfinite(b)) {
                    const uint64_t key = make_key(b, 0xFFFFFFFFu);  // below every real key of value b
                    if (publish && lane == 0 && gthr)
                        atomicMax(reinterpret_cast<unsigned long long*>(gthr) + n0 + i, static_cast<unsigned long long>(key));
                    g = key > g ? key : g;
                }
            }
            if (lane == 0) e.gcache[i] = g;
        }
    }
    if (etid < 2) e.more[etid] = 0;
    for (int i = etid; i < 4 * NG; i += nthr) e.mref[i] = -INFINITY;
}

// Appends, for every node j whose bit is set in `offer`, this lane's key
// key(z[j], row) to node j's candidate slots; returns the bits of the keys
// that found no free slot (offered again after the next merge).
__device__ __forceinline__ uint32_t epi_offer(const EpiSmem& e, int c0, const float (&z)[16], uint32_t offer,
                                              uint32_t row, int lane) {
    uint32_t pend = 0;
    if (__any_sync(kFull, offer != 0u)) {
#pragma unroll
        for (int j = 0; j < 16; j++) {
            const bool pass = (offer >> j) & 1u;
            const unsigned bal = __ballot_sync(kFull, pass);
            if (bal) {
                int base = 0;
                if (lane == 0) base = atomicAdd(&e.cnt[c0 + j], __popc(bal));
                base = __shfl_sync(kFull, base, 0);
                const int pos = base + __popc(bal & ((1u << lane) - 1u));
                if (pass) {
                    if (pos < e.cap)
                        e.cand[(c0 + j) * e.cap + pos] = make_key(z[j], row);
                    else
                        pend |= 1u << j;
                }
            }
        }
    }
    return pend;
}

// The subset of `pend` whose keys still beat their node's (raised)
// threshold (a threshold read before its update is lower: a superset).
__device__ __forceinline__ uint32_t epi_still_pass(const EpiSmem& e, int k, int c0, const float (&z)[16],
                                                   uint32_t pend, uint32_t row) {
    (void)k;
    uint32_t keep = 0;
#pragma unroll
    for (int j = 0; j < 16; j++)
        if (((pend >> j) & 1u) && make_key(z[j], row) > e.gcache[c0 + j]) keep |= 1u << j;
    return keep;
}

// One 16-node chunk of this thread's row (all 32 lanes, same chunk).
// ew: the warp's row quarter (0..3; per-quarter reference maxima and sums).
// z[j]: scaled logit of node c0+j of the group; node j exists iff bit j of
// nodemask is set; rowvalid: the row is < V.  ssum: the running sum of this
// lane's node (c0 + lane/2).  Returns the bits of the candidates that found
// no free slot (only possible when e.cap < the tile's rows).
__device__ __forceinline__ uint32_t epi_chunk(const EpiSmem& e, int NG, int k, int ew, int lane, int c0,
                                          float (&z)[16], uint32_t nodemask, bool rowvalid, uint32_t row,
                                          float& ssum) {
    bool ok[16];
#pragma unroll
    for (int j = 0; j < 16; j++) {
        ok[j] = rowvalid && ((nodemask >> j) & 1u);
        if (!ok[j]) z[j] = -INFINITY;
        else if (z[j] == 0.0f) z[j] = 0.0f;  // -0 -> +0
    }
    float* mr = e.mref + ew * NG + c0;
    float m[16];
#pragma unroll
    for (int j = 0; j < 16; j++) m[j] = mr[j];
    bool slow = false;
#pragma unroll
    for (int j = 0; j < 16; j++) slow |= z[j] > m[j] + kRefSlack;
    if (__any_sync(kFull, slow)) {
        const float mx = bfly16<true>(z, lane);
        const int me = lane >> 1;
        const float old = mr[me];
        const float nm = fmaxf(old, mx);
        if (old != -INFINITY && nm > old) ssum *= __expf(old - nm);
        __syncwarp();
        if ((lane & 1) == 0) mr[me] = nm;
        __syncwarp();
#pragma unroll
        for (int j = 0; j < 16; j++) m[j] = mr[j];
    }
    float p[16];
#pragma unroll
    for (int j = 0; j < 16; j++) p[j] = z[j] != -INFINITY ? __expf(z[j] - m[j]) : 0.0f;
    ssum += bfly16<false>(p, lane);
    uint32_t passmask = 0;  // bit j: this row's key beats node j's current threshold
#pragma unroll
    for (int j = 0; j < 16; j++)
        if (ok[j] && make_key(z[j], row) > e.gcache[c0 + j]) passmask |= 1u << j;
    return epi_offer(e, c0, z, passmask, row, lane);
}

__device__ __forceinline__ uint64_t shfl_u64(uint64_t v, int src) {
    const uint32_t lo = __shfl_sync(kFull, static_cast<uint32_t>(v), src);
    const uint32_t hi = __shfl_sync(kFull, static_cast<uint32_t>(v >> 32), src);
    return (static_cast<uint64_t>(hi) << 32) | lo;
}
__device__ __forceinline__ uint64_t shfl_xor_u64(uint64_t v, int m) {
    const uint32_t lo = __shfl_xor_sync(kFull, static_cast<uint32_t>(v), m);
    const uint32_t hi = __shfl_xor_sync(kFull, static_cast<uint32_t>(v >> 32), m);
    return (static_cast<uint64_t>(hi) << 32) | lo;
}
__device__ __forceinline__ uint64_t shfl_up_u64(uint64_t v, int dlt) {
    const uint32_t lo = __shfl_up_sync(kFull, static_cast<uint32_t>(v), dlt);
    const uint32_t hi = __shfl_up_sync(kFull, static_cast<uint32_t>(v >> 32), dlt);
    return (static_cast<uint64_t>(hi) << 32) | lo;
}

// Merges the c candidate keys C[0..c) into the sorted list L[0..k) (k <= 64)
// with one warp.  Keys are distinct; 0 marks empty slots.
__device__ __forceinline__ void warp_merge(uint64_t* L, const uint64_t* C, int c, int k, int lane) {
    if (c <= 4) {
        // few candidates: insert one at a time into the register-held list
        uint64_t a0 = lane < k ? L[lane] : 0ull;
        uint64_t a1 = lane + 32 < k ? L[lane + 32] : 0ull;
        for (int i = 0; i < c; i++) {
            const uint64_t x = C[i];
            const int p = __popc(__ballot_sync(kFull, a0 > x)) + __popc(__ballot_sync(kFull, a1 > x));
            if (p >= k) continue;
            const uint64_t u0 = shfl_up_u64(a0, 1), u1 = shfl_up_u64(a1, 1), l0 = shfl_u64(a0, 31);
            const uint64_t n0 = lane > p ? u0 : (lane == p ? x : a0);
            const uint64_t n1 = lane + 32 > p ? (lane == 0 ? l0 : u1) : (lane + 32 == p ? x : a1);
            a0 = n0;
            a1 = n1;
        }
        __syncwarp();
        if (lane < k) L[lane] = a0;
        if (lane + 32 < k) L[lane + 32] = a1;
        __syncwarp();
        return;
    }
    for (int b = 0; b < c; b += 32) {
        const int nb = min(32, c - b);
        uint64_t x = lane < nb ? C[b + lane] : 0ull;
        // bitonic sort of the batch, descending across lanes
#pragma unroll
        for (int size = 2; size <= 32; size <<= 1) {
#pragma unroll
            for (int stride = size >> 1; stride > 0; stride >>= 1) {
                const uint64_t y = shfl_xor_u64(x, stride);
                const bool desc_block = (lane & size) == 0;
                const bool lower = (lane & stride) == 0;
                const bool keep_max = lower == desc_block;
                x = keep_max ? (x > y ? x : y) : (x < y ? x : y);
            }
        }
        // new position of the batch element = #{list > x} + its rank in the batch
        int lo = 0, hi = k;
        while (lo < hi) {
            const int mid = (lo + hi) >> 1;
            if (L[mid] > x)
                lo = mid + 1;
            else
                hi = mid;
        }
        const int posx = lo + lane;
        // new position of a list element = old position + #{batch > element}
        uint64_t ent[2];
        int posn[2];
#pragma unroll
        for (int t = 0; t < 2; t++) {
            const int pos = lane + 32 * t;
            ent[t] = pos < k ? L[pos] : 0ull;
            int l2 = 0, h2 = 32;
#pragma unroll
            for (int it = 0; it < 6; it++) {
                const int mid = (l2 + h2) >> 1;
                const uint64_t bm = shfl_u64(x, mid & 31);
                if (l2 < h2) {
                    if (bm > ent[t])
                        l2 = mid + 1;
                    else
                        h2 = mid;
                }
            }
            posn[t] = pos + l2;
        }
        __syncwarp();
        if (posx < k && x != 0ull) L[posx] = x;
#pragma unroll
        for (int t = 0; t < 2; t++)
            if (lane + 32 * t < k && posn[t] < k) L[posn[t]] = ent[t];
        __syncwarp();
    }
}

// Merges every node's tile candidates into its list: one warp per node, no
// block barrier between nodes.  Called by all nthr epilogue threads; wi is
// the epilogue warp index (0 .. nthr/32 - 1).
//
// Cross-CTA filter: gthr[n] (global, zeroed before the launch) holds the
// largest k-th key any CTA has published for node n.  A CTA holding k keys
// >= b proves that no key <= b can be among the node's k best children of
// the whole vocabulary, so candidates must beat max(own k-th key, gthr[n]);
// keys are distinct, so the test is exact.  Each merge publishes the CTA's
// k-th key (atomicMax) and fetches gthr[n] for the next tile's filter.
__device__ __forceinline__ void epi_merge(const EpiSmem& e, int NG, int k, int wi, int lane, int nthr, int etid,
                                          uint64_t* gthr, int n0, int N, int* reset_flag = nullptr) {
    named_bar_sync(kEpiBarrier, nthr);
    if (reset_flag && etid == 0) *reset_flag = 0;  // every thread read it before this barrier
    uint64_t g = 0ull;
    if (gthr && etid < NG && n0 + etid < N) g = __ldcg(reinterpret_cast<const unsigned long long*>(gthr) + n0 + etid);
    for (int nd = wi; nd < NG; nd += nthr / 32) {
        const int c = min(e.cnt[nd], e.cap);
        if (c == 0) continue;
        warp_merge(e.list + nd * k, e.cand + nd * e.cap, c, k, lane);
        if (lane == 0) {
            e.cnt[nd] = 0;
            const uint64_t kth = e.list[nd * k + k - 1];
            if (gthr && kth != 0ull && n0 + nd < N)
                atomicMax(reinterpret_cast<unsigned long long*>(gthr) + n0 + nd, static_cast<unsigned long long>(kth));
        }
    }
    named_bar_sync(kEpiBarrier, nthr);
    // the filter threshold of the next tile (read after its first barrier):
    // the larger of the node's own k-th key and the cross-CTA bound
    if (etid < NG) {
        const uint64_t l = e.list[etid * k + k - 1];
        e.gcache[etid] = l > g ? l : g;
    }
}

// Records this warp's (reference, sum) of chunk cc's nodes.
__device__ __forceinline__ void epi_stash(const EpiSmem& e, int NG, int ew, int lane, int c0, float ssum) {
    if ((lane & 1) == 0) {
        const int nd = c0 + (lane >> 1);
        e.stats[ew * NG + nd] = make_float2(e.mref[ew * NG + nd], ssum);
    }
}

// Keys per node in the partial buffer: nV*k rounded up to even, so every
// node's block starts on a 16-byte boundary (it is read with 16-byte loads).
__host__ __device__ __forceinline__ int part_stride(int nV, int k) { return (nV * k + 1) & ~1; }

// Writes this CTA's partial results for the nodes n0 .. n0+NG-1 (< N), node
// major so that each node's partials are contiguous:
// part_ms[n][vr] = (max, sum exp), part_key[n * part_stride + vr*k + j] = top-k keys.
__device__ __forceinline__ void epi_finalize(const EpiSmem& e, int NG, int k, int etid, int nthr, int n0, int N,
                                             int vr, int nV, float2* part_ms, uint64_t* part_key) {
    named_bar_sync(kEpiBarrier, nthr);
    for (int c = etid; c < NG; c += nthr) {
        const int n = n0 + c;
        if (n >= N) continue;
        float2 a = e.stats[c];
        for (int w = 1; w < 4; w++) a = lse_merge(a, e.stats[w * NG + c]);
        part_ms[static_cast<size_t>(n) * nV + vr] = a;
    }
    for (int i = etid; i < NG * k; i += nthr) {
        const int c = i / k, j = i % k, n = n0 + c;
        if (n >= N) continue;
        part_key[static_cast<size_t>(n) * part_stride(nV, k) + static_cast<size_t>(vr) * k + j] = e.list[i];
    }
}

}  // namespace dart
