// Selection, emission and small elementwise kernels of the DARTree path.
//
//   merge_select  (Algorithm 1, scoring + "retain the global top-W"):
//       one block per expanded node merges the LM-head kernel's per-CTA
//       partials into log-sum-exp and the node's top-k children,
//       log q~ = min(z - lse, 0); the last block of each sequence (atomic
//       ticket, no waiting) then scores the candidates with Eq. 5 and keeps
//       the top-W as S_d.
//   prune_emit    (Algorithm 1 final step + Lemma 1, Sec. 2.3 flattening):
//       one block per sequence: global top-B by (score desc, node id asc),
//       compaction in id order, parent remap, depths, position ids and the
//       ancestor bit mask.
//   prep / gather / silu / residual_norm: the elementwise parts of the
//       fallback correction head around the two GEMMs.
#include "dart_device.cuh"
#include "dart_kernels.h"

namespace dart {

namespace {

constexpr int kSelThreads = 256;
constexpr int kEmitThreads = 1024;

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

// Selects the kk largest nonzero keys (kk >= 1, at least kk nonzero keys
// present) and writes them in descending order to out[0..kk).
__device__ __forceinline__ void block_topk_sorted(const uint64_t* keys, int n, int kk, uint64_t* out,
                                                  uint64_t* sel, uint32_t* hist, int* scal) {
    const uint64_t kth = block_kth_largest(keys, n, kk, hist, scal);
    if (threadIdx.x == 0) scal[2] = 0;
    __syncthreads();
    for (int i = threadIdx.x; i < n; i += blockDim.x) {
        const uint64_t x = keys[i];
        if (x != 0ull && x >= kth) sel[atomicAdd(&scal[2], 1)] = x;
    }
    __syncthreads();
    for (int i = threadIdx.x; i < kk; i += blockDim.x) {
        const uint64_t x = sel[i];
        int r = 0;
        for (int j = 0; j < kk; j++) r += sel[j] > x;
        out[r] = x;
    }
    __syncthreads();
}

__global__ void __launch_bounds__(kSelThreads) merge_select_kernel(const SelectArgs a) {
    extern __shared__ uint64_t keys[];  // max(nV*k, W*k) keys, then 2 x 64 selection slots
    __shared__ uint32_t hist[256];
    __shared__ int scal[4];
    __shared__ float redf[32];
    __shared__ float redm[32];
    __shared__ int redi[32];
    __shared__ int ticket;
    const int cap = max(a.nV * a.k, a.W * a.k);
    uint64_t* sel = keys + cap;
    uint64_t* top = sel + 64;

    const int n = blockIdx.x, tid = threadIdx.x;
    const int s = n / a.P, p = n % a.P;
    const int prev_count = a.dep == 1 ? 1 : a.tree_count[s * a.L + a.dep - 2];

    if (p < prev_count) {
        // log-sum-exp of the node's scaled logits from the per-CTA partials
        float2 acc = make_float2(-INFINITY, 0.0f);
        for (int r = tid; r < a.nV; r += kSelThreads) acc = lse_merge(acc, a.part_ms[static_cast<size_t>(r) * a.N + n]);
        const float gm = [&] {
            float m = warp_max(acc.x);
            if ((tid & 31) == 0) redm[tid >> 5] = m;
            __syncthreads();
            float t = -INFINITY;
            for (int i = 0; i < kSelThreads / 32; i++) t = fmaxf(t, redm[i]);
            return t;
        }();
        const float part = acc.x == -INFINITY ? 0.0f : acc.y * __expf(acc.x - gm);
        const float ssum = block_sum_float(part, redf);
        const float lse = gm == -INFINITY ? -INFINITY : gm + logf(ssum);
        // top-k over every CTA's top-k
        const int nk = a.nV * a.k;
        for (int i = tid; i < nk; i += kSelThreads) {
            const int r = i / a.k, j = i % a.k;
            keys[i] = a.part_key[(static_cast<size_t>(r) * a.N + n) * a.k + j];
        }
        __syncthreads();
        block_topk_sorted(keys, nk, a.k, top, sel, hist, scal);
        for (int j = tid; j < a.k; j += kSelThreads) {
            const uint64_t x = top[j];
            const float z = key_val(x);
            float lq = -INFINITY;
            if (lse != -INFINITY && z != -INFINITY) lq = fminf(z - lse, 0.0f);
            a.node_logq[static_cast<size_t>(n) * a.k + j] = lq;
            a.node_tok[static_cast<size_t>(n) * a.k + j] = static_cast<int>(key_idx(x));
        }
        if (tid == 0) a.node_lse[n] = lse;
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

    const int ncand = prev_count * a.k;
    int valid = 0;
    for (int c = tid; c < ncand; c += kSelThreads) {
        const int pp = c / a.k, j = c % a.k;
        const float ps = a.dep == 1 ? 0.0f : a.tree_score[(static_cast<size_t>(s) * a.L + a.dep - 2) * a.W + pp];
        const float lq = __ldcg(a.node_logq + static_cast<size_t>(s * a.P + pp) * a.k + j);
        const float sc = (ps + lq) + a.beta;  // Eq. 5, one more depth
        const bool ok = sc > -INFINITY;
        keys[c] = ok ? make_key(sc, static_cast<uint32_t>(c)) : 0ull;
        valid += ok;
    }
    const int nvalid = block_sum_int(valid, redi);
    const int cnt = min(a.W, nvalid);
    if (cnt > 0) block_topk_sorted(keys, ncand, cnt, top, sel, hist, scal);
    const size_t tb = (static_cast<size_t>(s) * a.L + a.dep - 1) * a.W;
    for (int r = tid; r < a.W; r += kSelThreads) {
        if (r < cnt) {
            const uint64_t x = top[r];
            const int c = static_cast<int>(key_idx(x));
            const int pp = c / a.k, j = c % a.k;
            const int tok = __ldcg(a.node_tok + static_cast<size_t>(s * a.P + pp) * a.k + j);
            a.tree_tok[tb + r] = tok;
            a.tree_parent[tb + r] = a.dep == 1 ? -1 : pp;
            a.tree_score[tb + r] = key_val(x);
            if (r < a.Pn) {
                a.child_prow[s * a.Pn + r] = s * a.P + pp;
                a.child_tok[s * a.Pn + r] = tok;
            }
        } else {
            a.tree_tok[tb + r] = -1;
            a.tree_parent[tb + r] = -1;
            a.tree_score[tb + r] = -INFINITY;
            if (r < a.Pn) {
                a.child_prow[s * a.Pn + r] = -1;
                a.child_tok[s * a.Pn + r] = 0;
            }
        }
    }
    if (tid == 0) a.tree_count[s * a.L + a.dep - 1] = cnt;
}

__global__ void __launch_bounds__(kEmitThreads) prune_emit_kernel(const EmitArgs a) {
    __shared__ uint64_t keys[1024];
    __shared__ int outidx[1024];
    __shared__ int par_out[1024];
    __shared__ uint32_t hist[256];
    __shared__ int scal[4];
    __shared__ int redi[32];
    __shared__ int wsum[32];
    const int s = blockIdx.x, tid = threadIdx.x;
    const int T = a.L * a.W;
    const size_t tb = static_cast<size_t>(s) * T;
    int valid = 0;
    if (tid < T) {
        const int dep = tid / a.W + 1, r = tid % a.W;
        const bool ok = r < a.tree_count[s * a.L + dep - 1];
        keys[tid] = ok ? make_key(a.tree_score[tb + tid], static_cast<uint32_t>(tid)) : 0ull;
        valid = ok;
    }
    const int nvalid = block_sum_int(valid, redi);
    const int beff = min(a.B, nvalid);
    uint64_t kth = ~0ull;
    if (beff > 0) kth = block_kth_largest(keys, T, beff, hist, scal);
    // compaction in ascending node id (exclusive scan of the selection flags)
    const int lane = tid & 31, warp = tid >> 5;
    const int flag = (tid < T && keys[tid] != 0ull && keys[tid] >= kth) ? 1 : 0;
    int incl = flag;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int t = __shfl_up_sync(0xFFFFFFFFu, incl, o);
        if (lane >= o) incl += t;
    }
    if (lane == 31) wsum[warp] = incl;
    __syncthreads();
    int base = 0;
    for (int i = 0; i < warp; i++) base += wsum[i];
    const int idx = base + incl - flag;
    if (tid < T) outidx[tid] = flag ? idx : -1;
    __syncthreads();
    const int B = a.B, nw = (B + 63) / 64;
    const size_t ob = static_cast<size_t>(s) * B;
    if (flag) {
        const int dep = tid / a.W + 1;
        int par = -1;
        if (dep > 1) {
            par = outidx[(dep - 2) * a.W + a.tree_parent[tb + tid]];
            if (par < 0) atomicOr(a.status, kDevOrphan);
        }
        par_out[idx] = par;
        a.tokens[ob + idx] = a.tree_tok[tb + tid];
        a.parents[ob + idx] = par;
        a.depths[ob + idx] = dep;
        a.pos_ids[ob + idx] = a.pos_offset + dep;
        a.scores[ob + idx] = a.tree_score[tb + tid];
    }
    __syncthreads();
    for (int i = beff + tid; i < B; i += kEmitThreads) {
        a.tokens[ob + i] = -1;
        a.parents[ob + i] = -2;
        a.depths[ob + i] = 0;
        a.pos_ids[ob + i] = -1;
        a.scores[ob + i] = -INFINITY;
    }
    // ancestor mask: bit j of row i set iff j is i or an ancestor of i
    for (int q = tid; q < B * nw; q += kEmitThreads) {
        const int i = q / nw, wd = q % nw;
        uint64_t word = 0ull;
        if (i < beff) {
            int j = i;
            while (j >= 0) {
                if ((j >> 6) == wd) word |= 1ull << (j & 63);
                j = par_out[j];
            }
        }
        a.mask[(ob + i) * nw + wd] = word;
    }
    if (tid == 0) a.n_nodes[s] = beff;
}

__device__ __forceinline__ void split_bf16(float x, __nv_bfloat16& hi, __nv_bfloat16& lo) {
    hi = __float2bfloat16_rn(x);
    lo = __float2bfloat16_rn(x - __bfloat162float(hi));
}

__global__ void prep_anchor_kernel(const float* anchor, int d, float* h, __nv_bfloat16* HL, int bhalf) {
    const int s = blockIdx.x;
    for (int j = threadIdx.x; j < d; j += blockDim.x) {
        const float x = anchor[static_cast<size_t>(s) * d + j];
        h[static_cast<size_t>(s) * d + j] = x;
        if (HL) {
            __nv_bfloat16 hi, lo;
            split_bf16(x, hi, lo);
            HL[static_cast<size_t>(s) * d + j] = hi;
            HL[static_cast<size_t>(bhalf + s) * d + j] = lo;
        }
    }
}

__global__ void gather_x_kernel(int d, const int* prow, const int* tok, const float* h, const void* E, int wbf16,
                                __nv_bfloat16* XL, int bhalf, float* X32) {
    const int c = blockIdx.x;
    const int pr = prow[c];
    const int t = tok[c];
    const size_t xo = static_cast<size_t>(c) * 2 * d;
    const size_t xl = static_cast<size_t>(bhalf + c) * 2 * d;
    for (int j = threadIdx.x; j < d; j += blockDim.x) {
        const float x = pr >= 0 ? h[static_cast<size_t>(pr) * d + j] : 0.0f;
        if (wbf16) {
            __nv_bfloat16 hi, lo;
            split_bf16(x, hi, lo);
            XL[xo + j] = hi;
            XL[xl + j] = lo;
            const __nv_bfloat16 ev = pr >= 0 ? reinterpret_cast<const __nv_bfloat16*>(E)[static_cast<size_t>(t) * d + j]
                                             : __float2bfloat16_rn(0.0f);
            XL[xo + d + j] = ev;
            XL[xl + d + j] = __float2bfloat16_rn(0.0f);
        } else {
            X32[xo + j] = x;
            X32[xo + d + j] = pr >= 0 ? reinterpret_cast<const float*>(E)[static_cast<size_t>(t) * d + j] : 0.0f;
        }
    }
}

__global__ void silu_split_kernel(int Nc, int d, int S, const float* part, __nv_bfloat16* AL, int bhalf, float* A32) {
    const size_t total = static_cast<size_t>(Nc) * d;
    for (size_t q = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; q < total;
         q += static_cast<size_t>(gridDim.x) * blockDim.x) {
        float u = 0.0f;
        for (int s = 0; s < S; s++) u += part[static_cast<size_t>(s) * total + q];
        const float act = u / (1.0f + expf(-u));
        if (AL) {
            __nv_bfloat16 hi, lo;
            split_bf16(act, hi, lo);
            AL[q] = hi;
            AL[static_cast<size_t>(bhalf) * d + q] = lo;
        } else {
            A32[q] = act;
        }
    }
}

__global__ void residual_norm_kernel(int d, int S, int Nc, const float* part, const int* prow, const float* h,
                                     float eps, float* h_next, __nv_bfloat16* HL, int bhalf) {
    __shared__ float red[32];
    const int c = blockIdx.x;
    const int pr = prow[c];
    const size_t total = static_cast<size_t>(Nc) * d;
    float ss = 0.0f;
    for (int i = threadIdx.x; i < d; i += blockDim.x) {
        float y = 0.0f;
        for (int s = 0; s < S; s++) y += part[static_cast<size_t>(s) * total + static_cast<size_t>(c) * d + i];
        const float r = pr >= 0 ? h[static_cast<size_t>(pr) * d + i] + y : 0.0f;
        h_next[static_cast<size_t>(c) * d + i] = r;
        ss += r * r;
    }
    const float tot = block_sum_float(ss, red);
    const float inv = 1.0f / sqrtf(tot / static_cast<float>(d) + eps);
    for (int i = threadIdx.x; i < d; i += blockDim.x) {
        const float x = h_next[static_cast<size_t>(c) * d + i] * inv;
        h_next[static_cast<size_t>(c) * d + i] = x;
        if (HL) {
            __nv_bfloat16 hi, lo;
            split_bf16(x, hi, lo);
            HL[static_cast<size_t>(c) * d + i] = hi;
            HL[static_cast<size_t>(bhalf + c) * d + i] = lo;
        }
    }
}

}  // namespace

int merge_select_smem(int nV, int k, int W) { return (max(nV * k, W * k) + 128) * 8; }

cudaError_t select_set_smem_limits(int max_dyn) {
    return cudaFuncSetAttribute(merge_select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, max_dyn);
}

cudaError_t launch_merge_select(const SelectArgs& a, cudaStream_t st) {
    const int smem = merge_select_smem(a.nV, a.k, a.W);
    merge_select_kernel<<<a.N, kSelThreads, smem, st>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_prune_emit(const EmitArgs& a, cudaStream_t st) {
    prune_emit_kernel<<<a.nseq, kEmitThreads, 0, st>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_prep_anchor(const float* anchor, int nseq, int d, float* h, __nv_bfloat16* HL, int bhalf,
                               cudaStream_t st) {
    prep_anchor_kernel<<<nseq, 256, 0, st>>>(anchor, d, h, HL, bhalf);
    return cudaGetLastError();
}

cudaError_t launch_gather_x(int Nc, int d, const int* prow, const int* tok, const float* h, const void* E,
                            int wbf16, __nv_bfloat16* XL, int bhalf, float* X32, cudaStream_t st) {
    gather_x_kernel<<<Nc, 256, 0, st>>>(d, prow, tok, h, E, wbf16, XL, bhalf, X32);
    return cudaGetLastError();
}

cudaError_t launch_silu_split(int Nc, int d, int S, const float* part, __nv_bfloat16* AL, int bhalf, float* A32,
                              cudaStream_t st) {
    const size_t total = static_cast<size_t>(Nc) * d;
    int blocks = static_cast<int>((total + 255) / 256);
    if (blocks > 4096) blocks = 4096;
    silu_split_kernel<<<blocks, 256, 0, st>>>(Nc, d, S, part, AL, bhalf, A32);
    return cudaGetLastError();
}

cudaError_t launch_residual_norm(int Nc, int d, int S, const float* part, const int* prow, const float* h,
                                 float eps, float* h_next, __nv_bfloat16* HL, int bhalf, cudaStream_t st) {
    residual_norm_kernel<<<Nc, 256, 0, st>>>(d, S, Nc, part, prow, h, eps, h_next, HL, bhalf);
    return cudaGetLastError();
}

}  // namespace dart
