// Seed scores of the starting bound of every node's top-k filter.
//
// Algorithm 1 scores every child of a node over the whole vocabulary and
// keeps the node's k best.  The LM-head kernel finds them by filtering: a
// logit is offered to the node's candidate lists only if its key beats a
// threshold that is a lower bound on the node's k-th best key.  Early in a
// vocabulary range that threshold is low (the first tile offers every
// logit), and at k >= 32 the list merges of those first tiles are what
// limits the kernel.
//
// Any set S of at least k rows bounds the k-th best score from below: the
// k-th largest score over S is at most the k-th largest over the whole
// vocabulary.  Here S holds, for each of R equal chunks of the vocabulary,
// the row with the largest drafter logit of the node's sequence at this
// depth (the drafter term dominates the score, so these rows hold most of
// the node's top-k).  This kernel recomputes each score over S in fp32 and
// lowers it by an error bound that covers both its own rounding and that of
// the LM-head (fp32 sums of d products of the bf16 row with the state's
// hi/lo split):
//     y = z~ - (2^-10 * max_i |E[r][i]| * sum_i |h[n][i]| * |1/T| + 2^-20 |z~|)
// so y <= z, the LM-head's score of that row.  The LM-head's epilogue warps
// (idle while the first tile streams in) take the k-th largest y of each
// node as the starting threshold of its filter and publish it as the node's
// bound for merge + select.  Keys below the node's k-th best are all that is
// ever skipped, so the result is unchanged.
#include "dart_device.cuh"
#include "dart_kernels.h"

namespace dart {

namespace {

constexpr int kBoundNodes = 8;  // nodes per block
constexpr int kBoundRows = 8;   // seed rows per block (one warp per row)

// Dynamic shared memory: E rows [8][d] bf16, states [8][d] fp32.
__global__ void __launch_bounds__(256) seed_score_kernel(const BoundArgs a) {
    pdl_trigger();
    extern __shared__ __align__(16) uint8_t sm_raw[];
    __nv_bfloat16* es = reinterpret_cast<__nv_bfloat16*>(sm_raw);
    float* hs = reinterpret_cast<float*>(sm_raw + static_cast<size_t>(kBoundRows) * a.d * 2);
    __shared__ __align__(8) uint64_t bar[2];
    __shared__ int rows[kBoundRows];
    __shared__ float hl1[kBoundNodes];
    __shared__ int abort_flag;
    const int nb = (a.P + kBoundNodes - 1) / kBoundNodes;
    const int s = blockIdx.x / nb, j0 = (blockIdx.x % nb) * kBoundNodes;
    const int nn = min(kBoundNodes, a.P - j0);
    const int n0 = s * a.P + j0;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int c = blockIdx.y * kBoundRows + warp;  // this warp's seed slot (vocabulary chunk)
    const int CH = (a.V + a.R - 1) / a.R;
    const float* dl = a.dlog + s * a.dlog_seq_stride + a.dlog_row_off;
    if (threadIdx.x == 0) {
        mbar_init(&bar[0], 1);
        mbar_init(&bar[1], 1);
        abort_flag = 0;
        fence_mbar_init();
    }

    // 1) the chunk's largest drafter logit (lowest row on ties); needs
    //    nothing of the previous kernel.  Sixteen independent loads per lane
    //    at a time: a chunk (~1200 rows at V = 151936) takes three L2 round
    //    trips instead of one per row of the lane.
    int r = -1;
    {
        float best = -INFINITY;
        const int v0 = c * CH, v1 = min(a.V, v0 + CH);
        for (int base = v0; base < v1; base += 32 * 16) {
            float x[16];
#pragma unroll
            for (int q = 0; q < 16; q++) {
                const int v = base + q * 32 + lane;
                x[q] = v < v1 ? __ldg(dl + v) : 0.0f;
            }
#pragma unroll
            for (int q = 0; q < 16; q++) {
                const int v = base + q * 32 + lane;
                if (v < v1 && (r < 0 || x[q] > best)) {
                    best = x[q];
                    r = v;
                }
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float ob = __shfl_xor_sync(kFull, best, o);
            const int orr = __shfl_xor_sync(kFull, r, o);
            if (orr >= 0 && (r < 0 || ob > best || (ob == best && orr < r))) {
                best = ob;
                r = orr;
            }
        }
    }
    if (lane == 0) rows[warp] = r;
    __syncthreads();
    const uint32_t ebytes = static_cast<uint32_t>(a.d) * 2, hbytes = static_cast<uint32_t>(a.d) * 4;
    int nrows = 0;
    for (int w = 0; w < kBoundRows; w++) nrows += rows[w] >= 0 ? 1 : 0;
    if (threadIdx.x == 0) {
        // the seed rows of E (the weights never depend on an earlier kernel)
        mbar_arrive_expect_tx(&bar[0], ebytes * nrows);
        for (int w = 0; w < kBoundRows; w++)
            if (rows[w] >= 0)
                bulk_load(es + static_cast<size_t>(w) * a.d, a.E + static_cast<size_t>(rows[w]) * a.d, ebytes, &bar[0]);
    }
    pdl_wait();
    if (threadIdx.x == 0) {
        mbar_arrive_expect_tx(&bar[1], hbytes * nn);
        for (int j = 0; j < nn; j++)
            bulk_load(hs + static_cast<size_t>(j) * a.d, a.h + static_cast<size_t>(n0 + j) * a.d, hbytes, &bar[1]);
    }
    volatile int* abort = &abort_flag;
    bool ok = mbar_wait(&bar[0], 0, abort) && mbar_wait(&bar[1], 0, abort);
    if (!ok) {
        *abort = 1;
        if (threadIdx.x == 0) atomicOr(a.status, kDevTimeout);
    }
    __syncthreads();
    if (*abort) {
        // no copy may still be in flight when the block exits
        if (threadIdx.x == 0) {
            const unsigned long long t0 = globaltimer_ns();
            while (!(mbar_try_wait(&bar[0], 0) && mbar_try_wait(&bar[1], 0)) && globaltimer_ns() - t0 < kWaitLimitNs) {
            }
        }
        __syncthreads();
        return;
    }

    // 2) sum_i |h[n][i]| of node warp
    if (warp < nn) {
        const float* hn = hs + static_cast<size_t>(warp) * a.d;
        float t = 0.0f;
        for (int i = lane * 4; i < a.d; i += 128) {
            const float4 q = *reinterpret_cast<const float4*>(hn + i);
            t += fabsf(q.x) + fabsf(q.y) + fabsf(q.z) + fabsf(q.w);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(kFull, t, o);
        if (lane == 0) hl1[warp] = t;
    }

    // 3) z~ of the block's 8 seed rows x 8 nodes: every thread a 8 x 8 block
    //    of partial sums over its slices of d (4 columns at
    //    (warp * 32 + lane) * 4 + 1024 m), so that each shared-memory value
    //    read feeds 8 products
    float acc[2][32];
#pragma unroll
    for (int q = 0; q < 64; q++) acc[q >> 5][q & 31] = 0.0f;
    float emax[kBoundRows];
#pragma unroll
    for (int rr = 0; rr < kBoundRows; rr++) emax[rr] = 0.0f;
    for (int i = (warp * 32 + lane) * 4; i < a.d; i += 1024) {
        float4 hv[kBoundNodes];
#pragma unroll
        for (int j = 0; j < kBoundNodes; j++)
            hv[j] = j < nn ? *reinterpret_cast<const float4*>(hs + static_cast<size_t>(j) * a.d + i)
                           : make_float4(0.0f, 0.0f, 0.0f, 0.0f);
#pragma unroll
        for (int rr = 0; rr < kBoundRows; rr++) {
            const uint2 u = *reinterpret_cast<const uint2*>(es + static_cast<size_t>(rr) * a.d + i);
            const float e0 = __uint_as_float(u.x << 16), e1 = __uint_as_float(u.x & 0xFFFF0000u);
            const float e2 = __uint_as_float(u.y << 16), e3 = __uint_as_float(u.y & 0xFFFF0000u);
            emax[rr] = fmaxf(emax[rr], fmaxf(fmaxf(fabsf(e0), fabsf(e1)), fmaxf(fabsf(e2), fabsf(e3))));
#pragma unroll
            for (int j = 0; j < kBoundNodes; j++) {
                const int q = rr * kBoundNodes + j;
                float t = acc[q >> 5][q & 31];
                t = fmaf(e0, hv[j].x, t);
                t = fmaf(e1, hv[j].y, t);
                t = fmaf(e2, hv[j].z, t);
                t = fmaf(e3, hv[j].w, t);
                acc[q >> 5][q & 31] = t;
            }
        }
    }
    // over the warp: lane l ends with the sums of outputs l and 32 + l;
    // then over the 8 warps in order (shared memory)
    warp_reduce_scatter32(acc[0], lane);
    warp_reduce_scatter32(acc[1], lane);
#pragma unroll
    for (int rr = 0; rr < kBoundRows; rr++) emax[rr] = warp_max(emax[rr]);
    __shared__ float red[8][64];
    __shared__ float remax[8][kBoundRows];
    red[warp][lane] = acc[0][0];
    red[warp][32 + lane] = acc[1][0];
    if (lane < kBoundRows) {
        float m = 0.0f;
#pragma unroll
        for (int rr = 0; rr < kBoundRows; rr++)
            if (lane == rr) m = emax[rr];
        remax[warp][lane] = m;
    }
    __syncthreads();  // red, remax, hl1
    if (threadIdx.x < kBoundRows * kBoundNodes) {
        const int rr = threadIdx.x / kBoundNodes, j = threadIdx.x % kBoundNodes;
        if (j < nn) {
            float dot = 0.0f, em = 0.0f;
#pragma unroll
            for (int w = 0; w < 8; w++) {
                dot += red[w][threadIdx.x];
                em = fmaxf(em, remax[w][rr]);
            }
            const int row = rows[rr];
            float y = -INFINITY;  // an empty chunk ranks last
            if (row >= 0) {
                const float z = (dot + __ldg(dl + row)) * a.invT;
                const float eps = ldexpf(em * hl1[j], -10) * fabsf(a.invT) + ldexpf(fabsf(z), -20);
                y = z == -INFINITY ? -INFINITY : z - eps;
                if (!(y == -INFINITY || isfinite(y))) y = __int_as_float(0x7FC00000);  // NaN: the node gets no bound
            }
            a.ybuf[static_cast<size_t>(n0 + j) * a.R + blockIdx.y * kBoundRows + rr] = y;
        }
    }
}

}  // namespace

cudaError_t launch_seed_score(const BoundArgs& a, int nseq, cudaStream_t st) {
    if (a.R <= 0 || a.R > kBoundMaxR || a.R % 32 != 0 || a.k < 1 || a.k > a.R || a.P < 1 || a.d % 8 != 0)
        return cudaErrorInvalidValue;
    const int nb = (a.P + kBoundNodes - 1) / kBoundNodes;
    return launch_pdl(seed_score_kernel, dim3(nseq * nb, a.R / kBoundRows), dim3(256), seed_score_smem(a.d), st, a);
}

size_t seed_score_smem(int d) { return static_cast<size_t>(kBoundRows) * d * 2 + static_cast<size_t>(kBoundNodes) * d * 4; }

// Dynamic shared memory allowed beside the kernel's static shared memory
// (set once to the device maximum, not to one plan's size).
cudaError_t seed_score_set_smem_limit(int smem_optin) {
    cudaFuncAttributes fa;
    cudaError_t e = cudaFuncGetAttributes(&fa, seed_score_kernel);
    if (e != cudaSuccess) return e;
    return cudaFuncSetAttribute(seed_score_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                smem_optin - static_cast<int>(fa.sharedSizeBytes));
}

int seed_score_static_smem() {
    cudaFuncAttributes fa;
    if (cudaFuncGetAttributes(&fa, seed_score_kernel) != cudaSuccess) return -1;
    return static_cast<int>(fa.sharedSizeBytes);
}

}  // namespace dart
