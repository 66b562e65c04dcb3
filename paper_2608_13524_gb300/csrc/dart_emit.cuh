// Prune and emit of one sequence (Algorithm 1 final step + Lemma 1, Sec. 3.3
// flattening): global top-B of the supertree by (score desc, node id asc),
// compaction in id order, parent remap, depths, position ids and the
// ancestor bit mask.  Called by every thread of a block of NT threads, one
// per supertree slot (L * W <= NT); used by the prune_emit kernel (one block
// per sequence) and by the fused small-problem round.
#pragma once

#include "dart_device.cuh"
#include "dart_kernels.h"

namespace dart {

// Number of keys > x in the descending list l[0..n) (binary search).
__device__ __forceinline__ int count_greater(const uint64_t* l, int n, uint64_t x) {
    int lo = 0, hi = n;
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (l[mid] > x)
            lo = mid + 1;
        else
            hi = mid;
    }
    return lo;
}

template <int NT>
__device__ __forceinline__ void prune_emit_seq(const EmitArgs& a, int s) {
    static_assert(NT <= 1024 && NT % 32 == 0, "one thread per supertree slot, at most 1024");
    __shared__ uint64_t keys[1024];
    __shared__ int outidx[1024];
    __shared__ int par_out[1024];
    __shared__ int cnts[1024];
    __shared__ int redi[32];
    __shared__ int wsum[32];
    const int tid = threadIdx.x;
    const int T = a.L * a.W;  // <= NT
    const size_t tb = static_cast<size_t>(s) * T;
    for (int dd = tid; dd < a.L; dd += NT) cnts[dd] = a.tree_count[s * a.L + dd];
    __syncthreads();
    int valid = 0;
    uint64_t my = 0ull;
    if (tid < T) {
        const int dep = tid / a.W + 1, r = tid % a.W;
        const bool ok = r < cnts[dep - 1];
        my = ok ? make_key(a.tree_score[tb + tid], static_cast<uint32_t>(tid)) : 0ull;
        keys[tid] = my;
        valid = ok;
    }
    const int nvalid = block_sum_int(valid, redi);  // synchronises: keys visible
    const int beff = min(a.B, nvalid);
    // Rank of a node = number of nodes with a larger key.  Each depth's list
    // is sorted (frontier rank order is score order, ties by id), so the rank
    // is a sum of L binary searches (Algorithm 1 final step: TopB by s_beta).
    int flag = 0;
    if (tid < T && my != 0ull) {
        int rank = 0;
        for (int dd = 0; dd < a.L; dd++) rank += count_greater(keys + dd * a.W, cnts[dd], my);
        flag = rank < beff;
    }
    // compaction in ascending node id (exclusive scan of the flags)
    const int lane = tid & 31, warp = tid >> 5;
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
            const int tp = a.tree_parent[tb + tid];
            if (bounds_check(a.status, tp >= 0 && tp < cnts[dep - 2])) par = outidx[(dep - 2) * a.W + tp];
            if (par < 0) atomicOr(a.status, kDevOrphan);
        }
        if (bounds_check(a.status, idx < beff)) {
            par_out[idx] = par;
            a.tokens[ob + idx] = a.tree_tok[tb + tid];
            a.parents[ob + idx] = par;
            a.depths[ob + idx] = dep;
            a.pos_ids[ob + idx] = a.pos_offset + dep;
            a.scores[ob + idx] = a.tree_score[tb + tid];
        }
    }
    __syncthreads();
    for (int i = beff + tid; i < B; i += NT) {
        a.tokens[ob + i] = -1;
        a.parents[ob + i] = -2;
        a.depths[ob + i] = 0;
        a.pos_ids[ob + i] = -1;
        a.scores[ob + i] = -INFINITY;
    }
    // ancestor mask: bit j of row i set iff j is i or an ancestor of i
    for (int q = tid; q < B * nw; q += NT) {
        const int i = q / nw, wd = q % nw;
        uint64_t word = 0ull;
        if (i < beff) {
            int j = i;
            while (j >= 0) {
                if (!bounds_check(a.status, j < beff)) break;
                if ((j >> 6) == wd) word |= 1ull << (j & 63);
                j = par_out[j];
            }
        }
        a.mask[(ob + i) * nw + wd] = word;
    }
    if (tid == 0) a.n_nodes[s] = beff;
}

}  // namespace dart
