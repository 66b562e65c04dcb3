// Best-first (heap-order) tree constructions that Table 2 of the paper
// compares DARTree with, on the GPU:
//
//   Domino-chain + DDTree   causal correction along ONE draft chain (the
//       depth-wise path with W = k = 1, which also writes each depth's
//       scaled logits), then DDTree (Sec. 3.3) over the chain-conditioned
//       distributions: the prefixes are scored with those position-wise
//       marginals, sum_i log q~_i(u_i) + beta d, and the best B are taken
//       best first.  ddtree_kernel runs the best-first search.
//   Sequential correction with heap   exact node-wise best-first search under
//       the corrected scores (Sec. 4.1): every pop corrects the popped prefix
//       (head update + scoring of its children) before the next pop.
//       seqheap_step_kernel performs one pop per sequence and prepares that
//       prefix's correction; the correction itself reuses the head-update,
//       LM-head, merge and top-K kernels.
//
// Both searches keep, for every popped node p (and the root), a cursor into
// its children sorted by log q~ (desc, token asc); p's "offer" is its best
// child not yet taken, scored s_p + log q~ + beta.  A pop takes the best offer
// by (score desc, node asc; the root first) -- DDTree's "next sibling / first
// child" pushes in another bookkeeping -- and the popped child becomes a node
// with its own offer.  Rows are emitted in pop order (parents first).
#include "dart_device.cuh"
#include "dart_kernels.h"

namespace dart {

namespace {

constexpr int kHeapThreads = 256;

// Key of an offer: score order, then the smaller slot (slot = node + 1, the
// root is slot 0).  An offer of score -inf is no offer (key 0).
__device__ __forceinline__ uint64_t offer_key(float v, int slot) {
    return v == -INFINITY ? 0ull : make_key(v, static_cast<uint32_t>(slot));
}

__device__ __forceinline__ uint64_t warp_max_u64(uint64_t v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const uint64_t y = shfl_xor_u64(v, o);
        v = y > v ? y : v;
    }
    return v;
}

// The best key among the offers of slots lane, lane + 32, ... < nslots.
__device__ __forceinline__ uint64_t lane_best(const float* offer, int nslots, int lane) {
    uint64_t b = 0ull;
    for (int o = lane; o < nslots; o += 32) {
        const uint64_t k = offer_key(offer[o], o);
        b = k > b ? k : b;
    }
    return b;
}

// Ancestor bit masks and padding of one sequence's emitted tree (rows in pop
// order, parents[] of its first n rows given).
__device__ void emit_masks(const int* par, int n, int B, size_t ob, int* tokens, int* parents, int* depths,
                           int* pos_ids, float* scores, uint64_t* mask) {
    const int nw = (B + 63) / 64;
    for (int i = n + static_cast<int>(threadIdx.x); i < B; i += blockDim.x) {
        tokens[ob + i] = -1;
        parents[ob + i] = -2;
        depths[ob + i] = 0;
        pos_ids[ob + i] = -1;
        scores[ob + i] = -INFINITY;
    }
    for (int q = threadIdx.x; q < B * nw; q += blockDim.x) {
        const int i = q / nw, wd = q % nw;
        uint64_t word = 0ull;
        if (i < n)
            for (int j = i; j >= 0; j = par[j])
                if ((j >> 6) == wd) word |= 1ull << (j & 63);
        mask[(ob + i) * nw + wd] = word;
    }
}

// One block per sequence.  Shared memory: the chain's sorted children per
// depth as log q~ [L][Bp] and tokens [L][Bp]; per popped node its parent,
// depth and score; per slot its cursor and offer.
__global__ void __launch_bounds__(kHeapThreads) ddtree_kernel(const DdtArgs a) {
    pdl_trigger();
    pdl_wait();
    extern __shared__ float hsm[];
    const int L = a.L, Bp = a.Bp, B = a.B;
    float* lq = hsm;                                          // [L][Bp]
    int* tk = reinterpret_cast<int*>(lq + L * Bp);            // [L][Bp]
    float* nsc = reinterpret_cast<float*>(tk + L * Bp);       // [B]
    int* npar = reinterpret_cast<int*>(nsc + B);              // [B]
    int* ndep = npar + B;                                     // [B]
    int* ntok = ndep + B;                                     // [B]
    int* next = ntok + B;                                     // [B + 1]
    float* offer = reinterpret_cast<float*>(next + B + 1);    // [B + 1]
    __shared__ int npop;
    const int s = blockIdx.x, tid = threadIdx.x, lane = tid & 31;
    // log q~ = min(z - lse, 0) of the chain's best Bp children per depth
    for (int q = tid; q < L * Bp; q += blockDim.x) {
        const int dd = q / Bp;
        const size_t src = (static_cast<size_t>(s) * L + dd) * Bp + (q % Bp);
        const float z = a.zval[src], lse = a.lse[static_cast<size_t>(s) * L + dd];
        lq[q] = (z == -INFINITY || lse == -INFINITY) ? -INFINITY : fminf(z - lse, 0.0f);
        tk[q] = a.tok[src];
    }
    __syncthreads();
    if (tid < 32) {
        // best-first search, one warp; lane l owns the slots l, l + 32, ...
        if (lane == 0) {
            next[0] = 0;
            offer[0] = Bp > 0 ? lq[0] + a.beta : -INFINITY;
        }
        __syncwarp();
        uint64_t best = lane == 0 ? offer_key(offer[0], 0) : 0ull;
        int n = 0;
        while (n < B) {
            const uint64_t k = warp_max_u64(best);
            if (k == 0ull) break;
            const int o = static_cast<int>(key_idx(k));
            const float sc = key_val(k);
            const int dep = o == 0 ? 1 : ndep[o - 1] + 1;
            if (lane == 0) {
                int c = next[o];
                if (!bounds_check(a.status, c < Bp && dep <= L)) c = 0;
                ntok[n] = tk[(dep - 1) * Bp + c];
                npar[n] = o - 1;
                ndep[n] = dep;
                nsc[n] = sc;
                next[o] = c + 1;
                const float so = o == 0 ? 0.0f : nsc[o - 1];
                offer[o] = c + 1 < Bp ? so + lq[(dep - 1) * Bp + c + 1] + a.beta : -INFINITY;
                next[n + 1] = 0;
                offer[n + 1] = (dep < L && Bp > 0) ? sc + lq[dep * Bp] + a.beta : -INFINITY;
            }
            __syncwarp();
            n++;
            if (lane == (o & 31)) best = lane_best(offer, n + 1, lane);
            else if (lane == (n & 31)) {
                const uint64_t kn = offer_key(offer[n], n);
                best = kn > best ? kn : best;
            }
        }
        if (lane == 0) npop = n;
    }
    __syncthreads();
    const int n = npop;
    const size_t ob = static_cast<size_t>(s) * B;
    for (int i = tid; i < n; i += blockDim.x) {
        a.tokens[ob + i] = ntok[i];
        a.parents[ob + i] = npar[i];
        a.depths[ob + i] = ndep[i];
        a.pos_ids[ob + i] = a.pos_offset + ndep[i];
        a.scores[ob + i] = nsc[i];
    }
    emit_masks(npar, n, B, ob, a.tokens, a.parents, a.depths, a.pos_ids, a.scores, a.mask);
    if (tid == 0) a.n_nodes[s] = n;
}

// One pop of the sequential search, one block per sequence (step t pops row
// t).  First the node popped at step t-1 is completed: if it was corrected,
// its state (the head update's output row s) is stored in its table slot and
// its offer is set from its sorted children (written by the top-K kernel at
// step t-1).  Then the best offer is popped, written as output row t, its
// parent's cursor advanced, and the new prefix's correction prepared: the
// parent's state as row s of the head's input (fp32, and as hi/lo bf16 rows
// for the tensor-core GEMM), the token, and the drafter row of its children.
__global__ void __launch_bounds__(kHeapThreads) seqheap_step_kernel(const SeqHeapArgs a, int t) {
    pdl_trigger();
    pdl_wait();
    __shared__ int sh[4];  // popped?, parent slot, token, depth
    const int s = blockIdx.x, tid = threadIdx.x, lane = tid & 31;
    const int B = a.B, Bp = a.Bp, L = a.L, d = a.d;
    const int S1 = B + 1;
    int* next = a.next + static_cast<size_t>(s) * S1;
    float* offer = a.offer + static_cast<size_t>(s) * S1;
    const size_t ob = static_cast<size_t>(s) * B;
    int* npop = a.npop + s;
    if (t == 0) {
        // the root (slot 0): its state is the anchor; its children were
        // scored and sorted by the setup launches (LM-head, merge, top-K)
        float* dst = a.tab + static_cast<size_t>(s) * S1 * d;
        for (int j = tid * 4; j < d; j += blockDim.x * 4)
            *reinterpret_cast<float4*>(dst + j) = *reinterpret_cast<const float4*>(a.anchor + static_cast<size_t>(s) * d + j);
        if (tid == 0) {
            next[0] = 0;
            const float lse = a.llse[static_cast<size_t>(s) * S1];
            const float z0 = a.lz[static_cast<size_t>(s) * S1 * Bp];
            offer[0] = (Bp > 0 && z0 != -INFINITY && lse != -INFINITY) ? fminf(z0 - lse, 0.0f) + a.beta : -INFINITY;
            *npop = 0;
        }
        __syncthreads();
    } else {
        const int prev = t - 1;  // the node popped at the previous step, if any
        const bool popped = __ldcg(npop) == t;
        if (popped && a.depths[ob + prev] < L) {
            // store its state: row s of the head update's output
            const float* src = a.hout + static_cast<size_t>(s) * d;
            float* dst = a.tab + (static_cast<size_t>(s) * S1 + t) * d;
            for (int j = tid * 4; j < d; j += blockDim.x * 4)
                *reinterpret_cast<float4*>(dst + j) = *reinterpret_cast<const float4*>(src + j);
            if (tid == 0) {
                const size_t lb = (static_cast<size_t>(s) * S1 + t);
                const float lse = a.llse[lb];
                const float z0 = a.lz[lb * Bp];
                next[t] = 0;
                offer[t] = (Bp > 0 && z0 != -INFINITY && lse != -INFINITY)
                               ? a.scores[ob + prev] + fminf(z0 - lse, 0.0f) + a.beta
                               : -INFINITY;
            }
        } else if (popped && tid == 0) {
            next[t] = 0;
            offer[t] = -INFINITY;  // a node at depth L has no children
        }
        __syncthreads();
    }
    if (tid < 32) {
        const int n = __ldcg(npop);
        uint64_t best = lane_best(offer, n + 1, lane);
        best = warp_max_u64(best);
        if (lane == 0) {
            sh[0] = 0;
            if (best != 0ull && n == t) {
                const int o = static_cast<int>(key_idx(best));
                const float sc = key_val(best);
                const size_t lb = static_cast<size_t>(s) * S1 + o;
                int c = next[o];
                const int dep = o == 0 ? 1 : a.depths[ob + o - 1] + 1;
                if (!bounds_check(a.status, c < Bp && o <= n && dep <= L)) c = 0;
                const int tok = a.ltok[lb * Bp + c];
                a.tokens[ob + n] = tok;
                a.parents[ob + n] = o - 1;
                a.depths[ob + n] = dep;
                a.pos_ids[ob + n] = a.pos_offset + dep;
                a.scores[ob + n] = sc;
                next[o] = c + 1;
                float so = 0.0f;
                if (o > 0) so = a.scores[ob + o - 1];
                const float z1 = c + 1 < Bp ? a.lz[lb * Bp + c + 1] : -INFINITY;
                const float lse = a.llse[lb];
                offer[o] = (z1 != -INFINITY && lse != -INFINITY) ? so + fminf(z1 - lse, 0.0f) + a.beta : -INFINITY;
                *npop = n + 1;
                sh[0] = 1;
                sh[1] = o;
                sh[2] = tok;
                sh[3] = dep;
            }
        }
    }
    __syncthreads();
    // the correction of the new prefix (a no-op input when nothing was popped)
    const int o = sh[0] ? sh[1] : 0;
    const float* src = a.tab + (static_cast<size_t>(s) * S1 + o) * d;
    for (int j = tid * 4; j < d; j += blockDim.x * 4) {
        const float4 v = *reinterpret_cast<const float4*>(src + j);
        *reinterpret_cast<float4*>(a.hin + static_cast<size_t>(s) * d + j) = v;
        if (a.HL) {
            __align__(8) __nv_bfloat16 hi[4], lo[4];
            split_bf16(v.x, hi[0], lo[0]);
            split_bf16(v.y, hi[1], lo[1]);
            split_bf16(v.z, hi[2], lo[2]);
            split_bf16(v.w, hi[3], lo[3]);
            *reinterpret_cast<uint2*>(a.HL + static_cast<size_t>(s) * d + j) = *reinterpret_cast<const uint2*>(hi);
            *reinterpret_cast<uint2*>(a.HL + static_cast<size_t>(a.bhalf + s) * d + j) =
                *reinterpret_cast<const uint2*>(lo);
        }
    }
    if (tid == 0) {
        a.child_prow[s] = s;
        a.child_tok[s] = sh[0] ? sh[2] : 0;
        a.dlog_row[s] = sh[0] ? min(sh[3], L - 1) : 0;
    }
}

// Masks and padding after the last pop.
__global__ void __launch_bounds__(kHeapThreads) seqheap_emit_kernel(const SeqHeapArgs a) {
    pdl_trigger();
    pdl_wait();
    const int s = blockIdx.x;
    const int n = __ldcg(a.npop + s);
    const size_t ob = static_cast<size_t>(s) * a.B;
    emit_masks(a.parents + ob, n, a.B, ob, a.tokens, a.parents, a.depths, a.pos_ids, a.scores, a.mask);
    if (threadIdx.x == 0) a.n_nodes[s] = n;
}

}  // namespace

int ddtree_smem(int L, int Bp, int B) { return (L * Bp * 2 + B * 4 + (B + 1) * 2) * 4; }

cudaError_t heap_set_smem_limits() { return set_max_dynamic_smem(reinterpret_cast<const void*>(ddtree_kernel)); }

cudaError_t launch_ddtree(const DdtArgs& a, cudaStream_t st) {
    return launch_pdl(ddtree_kernel, dim3(a.nseq), dim3(kHeapThreads), ddtree_smem(a.L, a.Bp, a.B), st, a);
}

cudaError_t launch_seqheap_step(const SeqHeapArgs& a, int t, cudaStream_t st) {
    return launch_pdl(seqheap_step_kernel, dim3(a.nseq), dim3(kHeapThreads), 0, st, a, t);
}

cudaError_t launch_seqheap_emit(const SeqHeapArgs& a, cudaStream_t st) {
    return launch_pdl(seqheap_emit_kernel, dim3(a.nseq), dim3(kHeapThreads), 0, st, a);
}

}  // namespace dart
