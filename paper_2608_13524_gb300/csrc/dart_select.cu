// Selection, emission and small elementwise kernels of the DARTree path.
//
//   merge_select  (Algorithm 1, scoring + "retain the global top-W"):
//       one block per expanded node merges the LM-head kernel's per-CTA
//       partials into log-sum-exp and the node's top-k children,
//       log q~ = min(z - lse, 0); the last block of each sequence (atomic
//       ticket, no waiting) then scores the candidates with Eq. 5 and keeps
//       the top-W as S_d.
//   prune_emit    (Algorithm 1 final step + Lemma 1, Sec. 3.3 flattening):
//       one block per sequence: global top-B by (score desc, node id asc),
//       compaction in id order, parent remap, depths, position ids and the
//       ancestor bit mask.
//   prep / gather / silu / gather_silu / residual_norm: the elementwise parts
//       of the fallback correction head around the two GEMMs (gather_silu
//       adds the per-token row of the split first layer's table).
#include <cstdlib>

#include "dart_device.cuh"
#include "dart_emit.cuh"
#include "dart_frontier.cuh"
#include "dart_kernels.h"

namespace dart {

namespace {

constexpr int kSelThreads = 512;
constexpr int kEmitThreads = 1024;

__global__ void __launch_bounds__(kSelThreads) merge_select_kernel(const SelectArgs a) {
    pdl_trigger();
    pdl_wait();
    // dynamic: max(nV*k, W*k) keys, kRankMax survivors, 64 outputs, W*k candidate tokens
    extern __shared__ uint64_t keys[];
    __shared__ uint32_t hist[256];
    __shared__ int scal[4];
    __shared__ uint64_t thr;
    __shared__ float redf[32];
    __shared__ float redm[32];
    __shared__ int redi[32];
    __shared__ int ticket;
    const int cap = max(a.nV * a.klist, a.W * a.k);
    uint64_t* surv = keys + cap;
    uint64_t* top = surv + kRankMax;
    int* ctok = reinterpret_cast<int*>(top + 64);

    const int n = blockIdx.x, tid = threadIdx.x;
    const int s = n / a.P, p = n % a.P;
    // this node's partials are contiguous: part_ms[n][nV], part_key[n][nV][klist];
    // they are loaded before the frontier size is known (rows past it hold
    // stale but harmless data)
    const int nk = a.nV * a.klist;
    const uint64_t* blk = a.part_key + static_cast<size_t>(n) * part_stride(a.nV, a.klist);  // 16-byte aligned
    const uint4* src = reinterpret_cast<const uint4*>(blk);
    const int prev_count = a.dep == 1 ? 1 : __ldcg(a.tree_count + s * a.L + a.dep - 2);
    const uint64_t bound = a.gthr ? __ldcg(reinterpret_cast<const unsigned long long*>(a.gthr) + n) : 0ull;
    float2 acc = make_float2(-INFINITY, 0.0f);
    {
        // every load of this thread is issued before the first use: one
        // L2 round trip instead of one per loop iteration
        constexpr int kBatch = 8;
        float2 ms[2];
#pragma unroll
        for (int u = 0; u < 2; u++) {
            const int r = tid + u * kSelThreads;
            ms[u] = r < a.nV ? __ldcg(a.part_ms + static_cast<size_t>(n) * a.nV + r) : make_float2(-INFINITY, 0.0f);
        }
        for (int r = tid + 2 * kSelThreads; r < a.nV; r += kSelThreads)
            acc = lse_merge(acc, __ldcg(a.part_ms + static_cast<size_t>(n) * a.nV + r));
        for (int i0 = 0; i0 < nk / 2; i0 += kBatch * kSelThreads) {
            uint4 v[kBatch];
#pragma unroll
            for (int u = 0; u < kBatch; u++) {
                const int i = i0 + u * kSelThreads + tid;
                if (i < nk / 2) v[u] = __ldcg(src + i);
            }
#pragma unroll
            for (int u = 0; u < kBatch; u++) {
                const int i = i0 + u * kSelThreads + tid;
                if (i < nk / 2) reinterpret_cast<uint4*>(keys)[i] = v[u];
            }
        }
        if ((nk & 1) && tid == 0) keys[nk - 1] = __ldcg(blk + nk - 1);
        acc = lse_merge(acc, ms[0]);
        acc = lse_merge(acc, ms[1]);
    }

    if (p < prev_count) {
        // log-sum-exp of the node's scaled logits from the per-CTA partials
        float m = warp_max(acc.x);
        if ((tid & 31) == 0) redm[tid >> 5] = m;
        __syncthreads();
        float gm = -INFINITY;
        for (int i = 0; i < kSelThreads / 32; i++) gm = fmaxf(gm, redm[i]);
        const float part = acc.x == -INFINITY ? 0.0f : acc.y * __expf(acc.x - gm);
        const float ssum = block_sum_float(part, redf);
        const float lse = gm == -INFINITY ? -INFINITY : gm + logf(ssum);
        // top-k over every CTA's (sorted) top-k list
        topk_of_sorted_lists(keys, a.nV, a.klist, a.k, bound, top, surv, &thr, hist, scal);
        for (int j = tid; j < a.k; j += kSelThreads) {
            const uint64_t x = top[j];
            const float z = key_val(x);
            float lq = -INFINITY;
            if (lse != -INFINITY && z != -INFINITY) lq = fminf(z - lse, 0.0f);
            a.node_logq[static_cast<size_t>(n) * a.k + j] = lq;
            a.node_tok[static_cast<size_t>(n) * a.k + j] = static_cast<int>(key_idx(x));
        }
        if (tid == 0) {
            a.node_lse[n] = lse;
            if (a.lse_hist) a.lse_hist[static_cast<size_t>(n) * a.lse_hist_stride] = lse;
        }
    } else {
        for (int j = tid; j < a.k; j += kSelThreads) {
            a.node_logq[static_cast<size_t>(n) * a.k + j] = -INFINITY;
            a.node_tok[static_cast<size_t>(n) * a.k + j] = -1;
        }
        if (tid == 0) a.node_lse[n] = -INFINITY;
    }

    // The last node block of this sequence selects S_d (no block ever waits).
    __threadfence();
    __syncthreads();
    if (tid == 0) ticket = atomicAdd(&a.seq_ticket[s], 1);
    __syncthreads();
    if (ticket != a.P - 1) return;
    __threadfence();
    if (tid == 0) a.seq_ticket[s] = 0;

    select_frontier(a, s, prev_count, keys, ctok, surv, top, &thr, hist, scal, redi);
}

__global__ void __launch_bounds__(kEmitThreads) prune_emit_kernel(const EmitArgs a) {
    pdl_trigger();
    pdl_wait();
    prune_emit_seq<kEmitThreads>(a, blockIdx.x);
}

// 4 consecutive floats -> 4 hi and 4 lo bf16 (8-byte stores)
__device__ __forceinline__ void split4(const float4 v, __nv_bfloat16* hi, __nv_bfloat16* lo) {
    __align__(8) __nv_bfloat16 h[4], l[4];
    split_bf16(v.x, h[0], l[0]);
    split_bf16(v.y, h[1], l[1]);
    split_bf16(v.z, h[2], l[2]);
    split_bf16(v.w, h[3], l[3]);
    *reinterpret_cast<uint2*>(hi) = *reinterpret_cast<const uint2*>(h);
    *reinterpret_cast<uint2*>(lo) = *reinterpret_cast<const uint2*>(l);
}

__global__ void prep_anchor_kernel(const float* anchor, int nseq, int d, float* h, __nv_bfloat16* HL, int bhalf,
                                   uint64_t* gthr_all, int n_gthr) {
    pdl_trigger();
    pdl_wait();
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n_gthr; i += gridDim.x * blockDim.x) gthr_all[i] = 0ull;
    const int q4 = d / 4;
    const int total = nseq * q4;
    for (int u = blockIdx.x * blockDim.x + threadIdx.x; u < total; u += gridDim.x * blockDim.x) {
        const int s = u / q4, j = (u % q4) * 4;
        const float4 x = *reinterpret_cast<const float4*>(anchor + static_cast<size_t>(s) * d + j);
        *reinterpret_cast<float4*>(h + static_cast<size_t>(s) * d + j) = x;
        if (HL) split4(x, HL + static_cast<size_t>(s) * d + j, HL + static_cast<size_t>(bhalf + s) * d + j);
    }
}

// X[c] = [h[prow[c]] ; E[tok[c]]]: one thread per 4 columns.
__global__ void gather_x_kernel(int Nc, int d, const int* prow, const int* tok, const float* h, const void* E,
                                int wbf16, __nv_bfloat16* XL, int bhalf, float* X32) {
    pdl_trigger();
    pdl_wait();
    const int q4 = (2 * d) / 4;
    const int total = Nc * q4;
    for (int u = blockIdx.x * blockDim.x + threadIdx.x; u < total; u += gridDim.x * blockDim.x) {
        const int c = u / q4, j = (u % q4) * 4;
        const int pr = prow[c];
        const size_t xo = static_cast<size_t>(c) * 2 * d + j;
        const size_t xl = static_cast<size_t>(bhalf + c) * 2 * d + j;
        if (j < d) {
            float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
            if (pr >= 0) x = *reinterpret_cast<const float4*>(h + static_cast<size_t>(pr) * d + j);
            if (wbf16)
                split4(x, XL + xo, XL + xl);
            else
                *reinterpret_cast<float4*>(X32 + xo) = x;
        } else {
            const size_t eo = static_cast<size_t>(tok[c]) * d + (j - d);
            if (wbf16) {
                uint2 e = make_uint2(0u, 0u);
                if (pr >= 0) e = *reinterpret_cast<const uint2*>(reinterpret_cast<const __nv_bfloat16*>(E) + eo);
                *reinterpret_cast<uint2*>(XL + xo) = e;
                *reinterpret_cast<uint2*>(XL + xl) = make_uint2(0u, 0u);
            } else {
                float4 e = make_float4(0.f, 0.f, 0.f, 0.f);
                if (pr >= 0) e = *reinterpret_cast<const float4*>(reinterpret_cast<const float*>(E) + eo);
                *reinterpret_cast<float4*>(X32 + xo) = e;
            }
        }
    }
}

// v += p[0] + p[stride] + ... (n terms, in this order), with up to 8 of the
// 16-byte loads in flight at once (a plain loop issues them one at a time).
__device__ __forceinline__ void add_splits(float4& v, const float* p, size_t stride, int n) {
    constexpr int kBatch = 8;
    for (int s0 = 0; s0 < n; s0 += kBatch) {
        float4 w[kBatch];
#pragma unroll
        for (int u = 0; u < kBatch; u++)
            if (s0 + u < n) w[u] = *reinterpret_cast<const float4*>(p + static_cast<size_t>(s0 + u) * stride);
#pragma unroll
        for (int u = 0; u < kBatch; u++) {
            if (s0 + u < n) {
                v.x += w[u].x;
                v.y += w[u].y;
                v.z += w[u].z;
                v.w += w[u].w;
            }
        }
    }
}

__global__ void silu_split_kernel(int Nc, int d, int S, const float* part, __nv_bfloat16* AL, int bhalf, float* A32) {
    pdl_trigger();
    pdl_wait();
    const size_t total = static_cast<size_t>(Nc) * d;
    const size_t t4 = total / 4;
    for (size_t u = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; u < t4;
         u += static_cast<size_t>(gridDim.x) * blockDim.x) {
        const size_t q = u * 4;
        float4 v = *reinterpret_cast<const float4*>(part + q);
        add_splits(v, part + total + q, total, S - 1);
        v.x = v.x / (1.0f + expf(-v.x));
        v.y = v.y / (1.0f + expf(-v.y));
        v.z = v.z / (1.0f + expf(-v.z));
        v.w = v.w / (1.0f + expf(-v.w));
        if (AL)
            split4(v, AL + q, AL + static_cast<size_t>(bhalf) * d + q);
        else
            *reinterpret_cast<float4*>(A32 + q) = v;
    }
}

// First head layer with the E half taken from the per-token table
// Q[t] = W_i[:, d:2d] . E[t] (computed once per handle):
//   a_c = SiLU(Q[tok[c]] + sum_s part[s][prow[c]]),
// where part holds the S k-split partials of W_i[:, 0:d] . h over the Np
// parents, then the hi/lo bf16 split of a_c (input of the W_o GEMM).  Empty
// child slots (prow < 0) and tokens outside [0, V) give a_c = 0.
__global__ void gather_silu_kernel(int Nc, int d, int S, int Np, const float* part, const int* prow, const int* tok,
                                   int V, const float* Q, __nv_bfloat16* AL, int bhalf, int* status) {
    pdl_trigger();
    pdl_wait();
    const size_t stride = static_cast<size_t>(Np) * d;
    const int q4 = d / 4;
    const int total = Nc * q4;
    for (int u = blockIdx.x * blockDim.x + threadIdx.x; u < total; u += gridDim.x * blockDim.x) {
        const int c = u / q4, j = (u % q4) * 4;
        int pr = prow[c];
        const int t = tok[c];
        if (pr >= 0 && !bounds_check(status, pr < Np && static_cast<unsigned>(t) < static_cast<unsigned>(V))) pr = -1;
        float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
        if (pr >= 0 && static_cast<unsigned>(t) < static_cast<unsigned>(V)) {
            v = *reinterpret_cast<const float4*>(Q + static_cast<size_t>(t) * d + j);
            add_splits(v, part + static_cast<size_t>(pr) * d + j, stride, S);
            v.x = v.x / (1.0f + expf(-v.x));
            v.y = v.y / (1.0f + expf(-v.y));
            v.z = v.z / (1.0f + expf(-v.z));
            v.w = v.w / (1.0f + expf(-v.w));
        }
        split4(v, AL + static_cast<size_t>(c) * d + j, AL + static_cast<size_t>(bhalf + c) * d + j);
    }
}

// One block per child: r = h[prow] + sum_s part[s], h_next = r / rms(r).
// NT = 1024 threads when S partial tiles are summed (many loads in flight),
// 256 for one summed tile (few registers, so blocks can become resident
// beside the GEMM before it ends).
template <int NT>
__global__ void __launch_bounds__(NT) residual_norm_kernel(int d, int S, int Nc, const float* part, const int* prow,
                                                           const float* h, float eps, float* h_next,
                                                           __nv_bfloat16* HL, int bhalf) {
    pdl_trigger();
    pdl_wait();
    __shared__ float red[32];
    const int c = blockIdx.x;
    const int pr = prow[c];
    const size_t total = static_cast<size_t>(Nc) * d;
    constexpr int kMaxPer = 16384 / (4 * NT);  // d <= 16384
    float4 r[kMaxPer];
    float ss = 0.0f;
#pragma unroll
    for (int it = 0; it < kMaxPer; it++) {
        const int j = (it * NT + threadIdx.x) * 4;
        r[it] = make_float4(0.f, 0.f, 0.f, 0.f);
        if (j < d && pr >= 0) {
            float4 v = *reinterpret_cast<const float4*>(h + static_cast<size_t>(pr) * d + j);
            add_splits(v, part + static_cast<size_t>(c) * d + j, total, S);
            r[it] = v;
            ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
        }
    }
    const float tot = block_sum_float(ss, red);
    const float inv = 1.0f / sqrtf(tot / static_cast<float>(d) + eps);
#pragma unroll
    for (int it = 0; it < kMaxPer; it++) {
        const int j = (it * NT + threadIdx.x) * 4;
        if (j < d) {
            const float4 v = make_float4(r[it].x * inv, r[it].y * inv, r[it].z * inv, r[it].w * inv);
            *reinterpret_cast<float4*>(h_next + static_cast<size_t>(c) * d + j) = v;
            if (HL) split4(v, HL + static_cast<size_t>(c) * d + j, HL + static_cast<size_t>(bhalf + c) * d + j);
        }
    }
}

}  // namespace

bool pdl_enabled() { return true; }

int merge_select_smem(int nV, int klist, int k, int W) {
    return (max(nV * klist, W * k) + kRankMax + 64) * 8 + W * k * 4;
}

cudaError_t select_set_smem_limits() { return set_max_dynamic_smem(reinterpret_cast<const void*>(merge_select_kernel)); }

cudaError_t launch_merge_select(const SelectArgs& a, cudaStream_t st) {
    const int smem = merge_select_smem(a.nV, a.klist, a.k, a.W);
    return launch_pdl(merge_select_kernel, dim3(a.N), dim3(kSelThreads), smem, st, a);
}

cudaError_t launch_prune_emit(const EmitArgs& a, cudaStream_t st) {
    return launch_pdl(prune_emit_kernel, dim3(a.nseq), dim3(kEmitThreads), 0, st, a);
}

static int grid_for(size_t units) {
    size_t b = (units + 255) / 256;
    return static_cast<int>(b < 1 ? 1 : (b > 2048 ? 2048 : b));
}

cudaError_t launch_prep_anchor(const float* anchor, int nseq, int d, float* h, __nv_bfloat16* HL, int bhalf,
                               uint64_t* gthr_all, int n_gthr, cudaStream_t st) {
    return launch_pdl(prep_anchor_kernel, dim3(grid_for(static_cast<size_t>(nseq) * d / 4)), dim3(256), 0, st, anchor,
                      nseq, d, h, HL, bhalf, gthr_all, n_gthr);
}

cudaError_t launch_gather_x(int Nc, int d, const int* prow, const int* tok, const float* h, const void* E,
                            int wbf16, __nv_bfloat16* XL, int bhalf, float* X32, cudaStream_t st) {
    return launch_pdl(gather_x_kernel, dim3(grid_for(static_cast<size_t>(Nc) * 2 * d / 4)), dim3(256), 0, st, Nc, d,
                      prow, tok, h, E, wbf16, XL, bhalf, X32);
}

cudaError_t launch_silu_split(int Nc, int d, int S, const float* part, __nv_bfloat16* AL, int bhalf, float* A32,
                              cudaStream_t st) {
    return launch_pdl(silu_split_kernel, dim3(grid_for(static_cast<size_t>(Nc) * d / 4)), dim3(256), 0, st, Nc, d, S,
                      part, AL, bhalf, A32);
}

cudaError_t launch_gather_silu(int Nc, int d, int S, int Np, const float* part, const int* prow, const int* tok,
                               int V, const float* Q, __nv_bfloat16* AL, int bhalf, int* status, cudaStream_t st) {
    return launch_pdl(gather_silu_kernel, dim3(grid_for(static_cast<size_t>(Nc) * d / 4)), dim3(256), 0, st, Nc, d, S,
                      Np, part, prow, tok, V, Q, AL, bhalf, status);
}

namespace {
// One thread evaluates one index check that fails (idx = n): the bounds bit
// is set in debug builds; nothing happens in release builds.  No memory but
// the status word is touched.
__global__ void bounds_probe_kernel(int* status, int idx, int n) { (void)bounds_check(status, idx < n); }
}  // namespace

cudaError_t launch_bounds_probe(int* status, cudaStream_t st) {
    bounds_probe_kernel<<<1, 1, 0, st>>>(status, 1, 1);
    return cudaGetLastError();
}

bool debug_build() {
#ifdef DART_DEBUG
    return true;
#else
    return false;
#endif
}

cudaError_t launch_residual_norm(int Nc, int d, int S, const float* part, const int* prow, const float* h,
                                 float eps, float* h_next, __nv_bfloat16* HL, int bhalf, cudaStream_t st) {
    if (S > 1)
        return launch_pdl(residual_norm_kernel<1024>, dim3(Nc), dim3(1024), 0, st, d, S, Nc, part, prow, h, eps,
                          h_next, HL, bhalf);
    return launch_pdl(residual_norm_kernel<256>, dim3(Nc), dim3(256), 0, st, d, S, Nc, part, prow, h, eps, h_next,
                      HL, bhalf);
}

}  // namespace dart
