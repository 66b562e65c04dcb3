// Frontier selection of one depth (Algorithm 1, "retain the global top-W"),
// shared by the selection kernels: the candidates (p, j) of sequence s are
// the k best children of each of its prev_count parents (node_logq /
// node_tok, rows s*P + p, each sorted by log q~), scored by Eq. 5,
// s = s_parent + log q~ + beta; the top W by (score desc, parent slot asc,
// rank asc) become S_dep.  Writes the supertree row of the depth, the child
// slots of the head update and the frontier count.  Every thread of the
// block calls it; keys / ctok hold W*k entries, surv kRankMax, top 64.
#pragma once

#include "dart_device.cuh"
#include "dart_kernels.h"

namespace dart {

__device__ __forceinline__ void select_frontier(const SelectArgs& a, int s, int prev_count, uint64_t* keys, int* ctok,
                                                uint64_t* surv, uint64_t* top, uint64_t* thr, uint32_t* hist,
                                                int* scal, int* redi) {
    const int tid = threadIdx.x;
    // candidates (p, j): parent p's list is sorted by log q~, hence by score
    const int ncand = prev_count * a.k;
    int valid = 0;
    for (int c = tid; c < ncand; c += static_cast<int>(blockDim.x)) {
        const int pp = c / a.k, j = c % a.k;
        const size_t src_i = static_cast<size_t>(s * a.P + pp) * a.k + j;
        const float ps = a.dep == 1 ? 0.0f : a.tree_score[(static_cast<size_t>(s) * a.L + a.dep - 2) * a.W + pp];
        const float lq = __ldcg(a.node_logq + src_i);
        ctok[c] = __ldcg(a.node_tok + src_i);
        const float sc = (ps + lq) + a.beta;  // Eq. 5, one more depth
        const bool ok = sc > -INFINITY;
        keys[c] = ok ? make_key(sc, static_cast<uint32_t>(c)) : 0ull;
        valid += ok;
    }
    const int nvalid = block_sum_int(valid, redi);
    const int cnt = min(a.W, nvalid);
    if (cnt > 0) topk_of_sorted_lists(keys, prev_count, a.k, cnt, 0ull, top, surv, thr, hist, scal);
    const size_t tb = (static_cast<size_t>(s) * a.L + a.dep - 1) * a.W;
    for (int r = tid; r < a.W; r += static_cast<int>(blockDim.x)) {
        if (r < cnt) {
            const uint64_t x = top[r];
            const int c = static_cast<int>(key_idx(x));
            if (!bounds_check(a.status, c < ncand)) continue;
            const int pp = c / a.k;
            const int tok = ctok[c];
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

}  // namespace dart
