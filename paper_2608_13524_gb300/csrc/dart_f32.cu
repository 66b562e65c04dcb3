// fp32 CUDA-core variants of the two contractions, for configurations whose
// weights are float32 (fp32 arithmetic throughout, no TF32).  They reuse the
// fused LM-head epilogue of dart_device.cuh, so the partial results have the
// same format as the tensor-core kernel's.
#include "dart_device.cuh"
#include "dart_kernels.h"

namespace dart {

namespace {

constexpr int kEPad = kBlockK + 1;  // padded row of the staged E tile (no bank conflicts)
constexpr int kEpiThreads = 128;    // 4 warps: thread r owns row r of a tile

// LM-head scoring, fp32: blocks of 128 threads (the 4 epilogue warps); thread
// r owns row r of each 128-row vocabulary tile.  CW node columns are computed
// (CW >= the node count: 4, 8 or 16 within a 16-node epilogue group, or 32).
// A vocabulary range is handled by a cluster of DS blocks that split the
// hidden dimension: each forms the partial dot products of its slice of d,
// and after a cluster barrier rank 0 adds the other ranks' partials from
// their shared memory in rank order (deterministic) and runs the fused
// epilogue alone.  DS > 1 only when there are fewer vocabulary tiles than
// SMs (small vocabularies), so the small problem still spreads over the GPU.
template <int NG, int CW>
__global__ void __launch_bounds__(kEpiThreads) lmhead_f32_kernel(const LmheadArgs a) {
    extern __shared__ float smf[];
    pdl_trigger();
    pdl_wait();
    float* Es = smf;                     // [128][65]
    float* Hs = Es + kTileM * kEPad;     // [CW][64]
    float* Ps = Hs + CW * kBlockK;       // [CW][128] this block's partial sums (DS > 1)
    EpiSmem e;
    e.cap = kCandCap;  // a whole tile: every candidate always fits
    e.list = reinterpret_cast<uint64_t*>(Ps + CW * kTileM);
    e.cand = e.list + NG * a.k;
    e.gcache = e.cand + NG * kCandCap;
    e.stats = reinterpret_cast<float2*>(e.gcache + NG);
    e.mref = reinterpret_cast<float*>(e.stats + 4 * NG);
    e.cnt = reinterpret_cast<int*>(e.mref + 4 * NG);
    e.more = e.cnt + NG;

    const int DS = a.DS;
    const int ds = DS > 1 ? static_cast<int>(cluster_ctarank()) : 0;
    const int cl = blockIdx.x / DS;
    const int g = cl % a.G;
    const int vr = cl / a.G;
    const int t0 = static_cast<int>((static_cast<long long>(vr) * a.tiles) / a.nV);
    const int t1 = static_cast<int>((static_cast<long long>(vr + 1) * a.tiles) / a.nV);
    const int tid = threadIdx.x, lane = tid & 31, ew = tid >> 5;
    const int KB = a.d / kBlockK;
    const int kb0 = ds * KB / DS, kb1 = (ds + 1) * KB / DS;
    if (ds == 0) epi_init(e, NG, a.k, tid, kEpiThreads);
    float ssum[NG / 16];
#pragma unroll
    for (int c = 0; c < NG / 16; c++) ssum[c] = 0.0f;

    for (int t = t0; t < t1; t++) {
        float acc[CW];
#pragma unroll
        for (int j = 0; j < CW; j++) acc[j] = 0.0f;
        for (int kb = kb0; kb < kb1; kb++) {
            named_bar_sync(kEpiBarrier, kEpiThreads);
            for (int q = tid; q < kTileM * (kBlockK / 4); q += kEpiThreads) {
                const int r = q / (kBlockK / 4), c4 = q % (kBlockK / 4);
                const int v = t * kTileM + r;
                float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
                if (v < a.V)
                    x = __ldg(reinterpret_cast<const float4*>(a.E32 + static_cast<size_t>(v) * a.d + kb * kBlockK) +
                              c4);
                float* dst = Es + r * kEPad + c4 * 4;
                dst[0] = x.x;
                dst[1] = x.y;
                dst[2] = x.z;
                dst[3] = x.w;
            }
            for (int q = tid; q < CW * kBlockK; q += kEpiThreads) {
                const int nn = q / kBlockK, c = q % kBlockK;
                const int n = g * NG + nn;
                Hs[q] = n < a.N ? a.h32[static_cast<size_t>(n) * a.d + kb * kBlockK + c] : 0.0f;
            }
            named_bar_sync(kEpiBarrier, kEpiThreads);
            const float* er = Es + tid * kEPad;
            for (int kk = 0; kk < kBlockK; kk++) {
                const float ev = er[kk];
#pragma unroll
                for (int j = 0; j < CW; j++) acc[j] = fmaf(ev, Hs[j * kBlockK + kk], acc[j]);
            }
        }
        if (DS > 1) {
            // sum the d-slices of the cluster on rank 0, in rank order
#pragma unroll
            for (int j = 0; j < CW; j++) Ps[j * kTileM + tid] = acc[j];
            cluster_sync_all();
            if (ds == 0)
                for (int r = 1; r < DS; r++) {
#pragma unroll
                    for (int j = 0; j < CW; j++)
                        acc[j] += ld_cluster_f32(smem_u32(Ps + j * kTileM + tid), static_cast<uint32_t>(r));
                }
            cluster_sync_all();  // the partials are read before any block overwrites them
        }
        if (ds != 0) continue;
        const int v = t * kTileM + tid;
        const bool valid = v < a.V;
        int cur_seq = -1;
        float dl = 0.0f;
#pragma unroll
        for (int c0 = 0; c0 < NG; c0 += 16) {
            float z[16];
            uint32_t nodemask = 0;
#pragma unroll
            for (int j = 0; j < 16; j++) {
                const int n = g * NG + c0 + j;
                z[j] = 0.0f;
                if (c0 + j < CW && n < a.N) {
                    nodemask |= 1u << j;
                    const int seq = n / a.P;
                    if (seq != cur_seq) {
                        cur_seq = seq;
                        const long long off = a.dlog_row ? static_cast<long long>(__ldg(a.dlog_row + seq)) * a.V
                                                         : a.dlog_row_off;
                        dl = valid ? __ldg(a.dlog + seq * a.dlog_seq_stride + off + v) : 0.0f;
                    }
                    z[j] = (acc[c0 + j < CW ? c0 + j : 0] + dl) * a.invT;
                    if (a.zout && valid) a.zout[static_cast<long long>(n) * a.zout_stride + v] = z[j];
                }
            }
            (void)epi_chunk(e, NG, a.k, ew, lane, c0, z, nodemask, valid, static_cast<uint32_t>(v), ssum[c0 / 16]);
        }
        epi_merge(e, NG, a.k, ew, lane, kEpiThreads, tid, a.gthr, g * NG, a.N);
    }
    if (ds != 0) return;
#pragma unroll
    for (int c0 = 0; c0 < NG; c0 += 16) epi_stash(e, NG, ew, lane, c0, ssum[c0 / 16]);
    epi_finalize(e, NG, a.k, tid, kEpiThreads, g * NG, a.N, vr, a.nV, a.part_ms, a.part_key);
}

// out[split][n][m] = sum_{k in split} A[m][k] * B[n][k]; 64 x 16 output tile
// per block of 256 threads, each thread 4 outputs.
constexpr int kGM = 64, kGN = 16, kGK = 32;

__global__ void __launch_bounds__(256) gemm_f32_kernel(const GemmArgs a) {
    __shared__ float As[kGM][kGK + 1];
    __shared__ float Bs[kGN][kGK + 1];
    pdl_trigger();
    pdl_wait();
    const int mt = blockIdx.x % a.MT;
    const int rest = blockIdx.x / a.MT;
    const int g = rest % a.G;
    const int split = rest / a.G;
    const int nchunk = a.K / kGK;
    const int c0 = static_cast<int>((static_cast<long long>(split) * nchunk) / a.S);
    const int c1 = static_cast<int>((static_cast<long long>(split + 1) * nchunk) / a.S);
    const int tid = threadIdx.x, tm = tid % kGM, tn = tid / kGM;
    const int m0 = mt * kGM;
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
    for (int c = c0; c < c1; c++) {
        for (int q = tid; q < kGM * kGK; q += 256) {
            const int r = q / kGK, kk = q % kGK;
            const int m = m0 + r;
            As[r][kk] = m < a.M ? a.A32[static_cast<size_t>(m) * a.K + c * kGK + kk] : 0.0f;
        }
        for (int q = tid; q < kGN * kGK; q += 256) {
            const int r = q / kGK, kk = q % kGK;
            const int n = g * kGN + r;
            Bs[r][kk] = n < a.N ? a.B32[static_cast<size_t>(n) * a.K + c * kGK + kk] : 0.0f;
        }
        __syncthreads();
#pragma unroll 8
        for (int kk = 0; kk < kGK; kk++) {
            const float av = As[tm][kk];
#pragma unroll
            for (int q = 0; q < 4; q++) acc[q] = fmaf(av, Bs[tn * 4 + q][kk], acc[q]);
        }
        __syncthreads();
    }
    const int m = m0 + tm;
    if (m < a.M) {
        float* out = a.out + static_cast<size_t>(split) * a.N * a.M;
#pragma unroll
        for (int q = 0; q < 4; q++) {
            const int n = g * kGN + tn * 4 + q;
            if (n < a.N) out[static_cast<size_t>(n) * a.M + m] = acc[q];
        }
    }
}

// The whole fallback-head update of one child per cluster, fp32, for small
// hidden sizes (d <= 1024): h_c = RMSNorm(h_p + W_o SiLU(W_i [h_p ; E[t_c]])).
// The S blocks of child c's cluster each own F = d / S output features: u
// and SiLU(u) of its features (W_i rows . [h_p ; E[t]]), then, once the
// cluster has all of SiLU(u) (read from the peers' shared memory), y = W_o
// rows . SiLU(u), r = h_p + y and the sum of r^2 of its features; the sums
// of the S blocks (rank order) give the RMS, and each block writes its
// normalised features.  One warp per feature, lanes over the dot product in
// a fixed order, so the result is deterministic.  This replaces the gather /
// W_i GEMM / SiLU / W_o GEMM / residual-norm launches of a depth.
constexpr int kHeadThreads = 256;

// sum_j w[j] * x[j] over n floats (n multiple of 4, both 16-byte aligned),
// by a group of g threads (a power of two dividing 32, consecutive lanes):
// thread `sub` takes the float4s sub, sub + g, ... (eight loads in flight),
// then the group adds its partials by a butterfly; every thread of the group
// returns the sum.  Fixed order: deterministic.
__device__ __forceinline__ float group_dot(const float* w, const float* x, int n, int g, int sub) {
    const float4* w4 = reinterpret_cast<const float4*>(w);
    const float4* x4 = reinterpret_cast<const float4*>(x);
    const int n4 = n / 4;
    float acc = 0.0f;
    for (int b = sub; b < n4; b += 8 * g) {
        float4 wv[8];
#pragma unroll
        for (int u = 0; u < 8; u++) wv[u] = b + u * g < n4 ? __ldg(w4 + b + u * g) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int u = 0; u < 8; u++) {
            if (b + u * g < n4) {
                const float4 xv = x4[b + u * g];
                acc = fmaf(wv[u].x, xv.x, acc);
                acc = fmaf(wv[u].y, xv.y, acc);
                acc = fmaf(wv[u].z, xv.z, acc);
                acc = fmaf(wv[u].w, xv.w, acc);
            }
        }
    }
    for (int o = g >> 1; o > 0; o >>= 1) acc += __shfl_xor_sync(0xFFFFFFFFu, acc, o);
    return acc;
}

// The whole fallback-head update of one child per cluster, fp32, for small
// hidden sizes (d <= 1024): h_c = RMSNorm(h_p + W_o SiLU(W_i [h_p ; E[t_c]])).
// The S blocks of child c's cluster each own F = d / S output features: u
// and SiLU(u) of its features (W_i rows . [h_p ; E[t]]), then, once the
// cluster has all of SiLU(u) (read from the peers' shared memory), y = W_o
// rows . SiLU(u), r = h_p + y and the sum of r^2 of its features; the sums
// of the S blocks (rank order) give the RMS, and each block writes its
// normalised features.  A group of 256 / F threads per feature, in a fixed
// order, so the result is deterministic.  This replaces the gather / W_i GEMM
// / SiLU / W_o GEMM / residual-norm launches of a depth.
__global__ void __launch_bounds__(kHeadThreads) head_small_f32_kernel(int d, int S, const int* prow, const int* tok,
                                                                      const float* h, const float* E,
                                                                      const float* Wi, const float* Wo, float eps,
                                                                      float* hnext) {
    extern __shared__ __align__(16) float hsm[];
    float* x = hsm;              // [2d]: h_p ; E[t]
    float* af = x + 2 * d;       // [d]: SiLU(u) of the whole child
    float* mine = af + d;        // [F]: SiLU(u) of this block's features
    float* rr = mine + d / S;    // [F]: r of this block's features
    __shared__ float ssq;
    pdl_trigger();
    pdl_wait();
    const int c = blockIdx.x / S;
    const uint32_t rank = cluster_ctarank();
    const int F = d / S, f0 = static_cast<int>(rank) * F;
    const int tid = threadIdx.x, lane = tid & 31;
    // threads per feature: the largest power of two <= 256 / F (and <= 32);
    // every thread runs every round (rows past F repeat feature 0, unused) so
    // that the group shuffles always see full warps
    int g = 1;
    while (g < 32 && 2 * g * F <= kHeadThreads) g *= 2;
    const int sub = lane & (g - 1);
    const int per_round = kHeadThreads / g;
    const int pr = prow[c], t = tok[c];
    for (int j = tid; j < d; j += kHeadThreads) {  // an empty child slot (pr < 0) gets a zero state
        x[j] = pr >= 0 ? h[static_cast<size_t>(pr) * d + j] : 0.0f;
        x[d + j] = E[static_cast<size_t>(t) * d + j];
    }
    __syncthreads();
    for (int base = 0; base < F; base += per_round) {
        const int f = base + tid / g;
        const bool ok = f < F;
        const float u = group_dot(Wi + static_cast<size_t>(f0 + (ok ? f : 0)) * 2 * d, x, 2 * d, g, sub);
        if (ok && sub == 0) mine[f] = u / (1.0f + __expf(-u));
    }
    cluster_sync_all();
    for (int j = tid; j < d; j += kHeadThreads)
        af[j] = ld_cluster_f32(smem_u32(mine + (j % F)), static_cast<uint32_t>(j / F));
    __syncthreads();
    for (int base = 0; base < F; base += per_round) {
        const int f = base + tid / g;
        const bool ok = f < F;
        const float y = group_dot(Wo + static_cast<size_t>(f0 + (ok ? f : 0)) * d, af, d, g, sub);
        if (ok && sub == 0) rr[f] = x[f0 + f] + y;
    }
    __syncthreads();
    if (tid < 32) {
        float part = 0.0f;
        for (int f = lane; f < F; f += 32) part = fmaf(rr[f], rr[f], part);
        for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(0xFFFFFFFFu, part, o);
        if (lane == 0) ssq = part;
    }
    cluster_sync_all();
    float tot = 0.0f;
    for (int q = 0; q < S; q++) tot += ld_cluster_f32(smem_u32(&ssq), static_cast<uint32_t>(q));
    const float inv = rsqrtf(tot / static_cast<float>(d) + eps);
    for (int f = tid; f < F; f += kHeadThreads) hnext[static_cast<size_t>(c) * d + f0 + f] = pr >= 0 ? rr[f] * inv : 0.0f;
    cluster_sync_all();  // peers finish reading this block's shared memory before it exits
}

template <int NG>
int smem_ng(int k, int CW) {
    return (kTileM * kEPad + CW * kBlockK + CW * kTileM) * 4 + NG * k * 8 + NG * kCandCap * 8 + NG * 8 + 4 * NG * 8 +
           4 * NG * 4 + NG * 4 + 8;
}

}  // namespace

int lmhead_f32_cw(int N) { return N <= 4 ? 4 : (N <= 8 ? 8 : (N <= 16 ? 16 : 32)); }

int lmhead_f32_smem(int NG, int k) {
    return NG <= 16 ? smem_ng<16>(k, 16) : smem_ng<32>(k, 32);  // the largest CW of the group size
}

cudaError_t f32_set_smem_limits(int max_dyn) {
    (void)max_dyn;
    cudaError_t e = cudaSuccess;
    for (const void* fn : {reinterpret_cast<const void*>(lmhead_f32_kernel<16, 4>),
                           reinterpret_cast<const void*>(lmhead_f32_kernel<16, 8>),
                           reinterpret_cast<const void*>(lmhead_f32_kernel<16, 16>),
                           reinterpret_cast<const void*>(lmhead_f32_kernel<32, 32>)})
        if (e == cudaSuccess) e = set_max_dynamic_smem(fn);
    return e;
}

cudaError_t launch_lmhead_f32(const LmheadArgs& a, cudaStream_t st) {
    const int smem = lmhead_f32_smem(a.NG, a.k);
    const dim3 grid(a.nV * a.G * a.DS);
    const int cw = a.NG == 16 ? lmhead_f32_cw(a.N) : 32;
    auto go = [&](auto kernel) {
        return a.DS > 1 ? launch_pdl_cluster(kernel, grid, dim3(kEpiThreads), smem, st, a.DS, a)
                        : launch_pdl(kernel, grid, dim3(kEpiThreads), smem, st, a);
    };
    if (a.NG == 16 && cw == 4) return go(lmhead_f32_kernel<16, 4>);
    if (a.NG == 16 && cw == 8) return go(lmhead_f32_kernel<16, 8>);
    if (a.NG == 16) return go(lmhead_f32_kernel<16, 16>);
    if (a.NG == 32) return go(lmhead_f32_kernel<32, 32>);
    return cudaErrorInvalidValue;
}

int head_small_f32_slices(int d) {
    if (d > 1024) return 0;
    int S = 8;
    while (S > 1 && (d % S != 0 || d / S < 32)) S /= 2;
    return S;
}

cudaError_t launch_head_small_f32(int Nc, int d, const int* prow, const int* tok, const float* h, const float* E,
                                  const float* Wi, const float* Wo, float eps, float* hnext, cudaStream_t st) {
    const int S = head_small_f32_slices(d);
    if (S == 0) return cudaErrorInvalidValue;
    const size_t smem = (static_cast<size_t>(3) * d + 2 * (d / S)) * 4;
    if (smem > 48 * 1024) {
        const cudaError_t e = set_max_dynamic_smem(reinterpret_cast<const void*>(head_small_f32_kernel));
        if (e != cudaSuccess) return e;
    }
    return launch_pdl_cluster(head_small_f32_kernel, dim3(Nc * S), dim3(kHeadThreads), smem, st, S, d, S, prow, tok,
                              h, E, Wi, Wo, eps, hnext);
}

cudaError_t launch_gemm_f32(const GemmArgs& a, cudaStream_t st) {
    return launch_pdl(gemm_f32_kernel, dim3(a.MT * a.G * a.S), dim3(256), 0, st, a);
}

}  // namespace dart
