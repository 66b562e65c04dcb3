// Candidate-restricted scoring (Algorithm 1 with a candidate-vocabulary size
// K > 0; the paper's default is K = 64):
//
//   cand_topk   C_d = TopK(L_d^base, K): for every (sequence, position) row
//               of the drafter logits, the K tokens with the largest base
//               logit (ties: token asc), written in ascending token order.
//               Once per round, for all L positions.
//   cand_score  for every node n of S_{d-1} and every candidate c of its
//               sequence's C_d: z = (Dlog[d-1][c] + E[c] . h_n) / T', in fp32
//               on CUDA cores (the dot products are K*N*d, far too small for
//               the tensor cores to matter).  Written in the LM-head's
//               partial format with one single-key list per candidate:
//               part_ms[n][i] = (z, 1), part_key[n][i] = key(z, c), so the
//               merge kernel computes log-sum-exp over C_d (q~ renormalised
//               over the candidates) and the node's top-k unchanged.
#include <algorithm>

#include "dart_device.cuh"
#include "dart_kernels.h"

namespace dart {

namespace {

constexpr int kTopkThreads = 1024;
constexpr int kDigitBits = 12;
constexpr int kBins = 1 << kDigitBits;  // histogram bins per radix pass
constexpr int kCollCap = 8192;          // keys of the threshold bin finished in shared memory (radix path)

// Returns, in lanes of warp 0, the largest digit b with
// sum_{b' >= b} hist[b'] >= need (need >= 1), and the count above b.
__device__ __forceinline__ void find_digit(const uint32_t* hist, int need, int* out) {
    const int lane = threadIdx.x & 31;
    constexpr int kPer = kBins / 32;
    // lane l owns bins [kBins - (l+1)*kPer, kBins - l*kPer), highest first
    uint32_t sum = 0;
    for (int j = 0; j < kPer; j++) sum += hist[kBins - 1 - lane * kPer - j];
    uint32_t incl = sum;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t t = __shfl_up_sync(0xFFFFFFFFu, incl, o);
        if (lane >= o) incl += t;
    }
    const unsigned hit = __ballot_sync(0xFFFFFFFFu, incl >= static_cast<uint32_t>(need));
    const int first = __ffs(hit) - 1;  // some lane always hits: the row holds >= need keys
    if (lane == first) {
        uint32_t cum = incl - sum;
        int b = kBins - 1 - lane * kPer;
        for (int j = 0; j < kPer; j++, b--) {
            const uint32_t c = hist[b];
            if (cum + c >= static_cast<uint32_t>(need)) break;
            cum += c;
        }
        out[0] = b;
        out[1] = static_cast<int>(cum);
    }
}

// Loads in flight per thread in the row passes (the row streams from HBM on
// the first pass; one load at a time would make it latency-bound).
constexpr int kRowBatch = 8;

// Calls f(value, token) for every element of this thread's strided share of
// the row, with kRowBatch 16-byte loads in flight when the row is 16-byte
// aligned (else 4-byte loads).
template <typename F>
__device__ __forceinline__ void for_row(const float* x, int V, F&& f) {
    const int tid = threadIdx.x;
    if ((V & 3) == 0 && (reinterpret_cast<uintptr_t>(x) & 15u) == 0) {
        const int V4 = V >> 2;
        const float4* x4 = reinterpret_cast<const float4*>(x);
        for (int q0 = tid; q0 < V4; q0 += kRowBatch * kTopkThreads) {
            float4 xs[kRowBatch];
#pragma unroll
            for (int u = 0; u < kRowBatch; u++) {
                const int q = q0 + u * kTopkThreads;
                xs[u] = q < V4 ? __ldg(x4 + q) : make_float4(0.f, 0.f, 0.f, 0.f);
            }
#pragma unroll
            for (int u = 0; u < kRowBatch; u++) {
                const int q = q0 + u * kTopkThreads;
                if (q < V4) {
                    f(xs[u].x, 4 * q);
                    f(xs[u].y, 4 * q + 1);
                    f(xs[u].z, 4 * q + 2);
                    f(xs[u].w, 4 * q + 3);
                }
            }
        }
    } else {
        for (int v0 = tid; v0 < V; v0 += 4 * kRowBatch * kTopkThreads) {
            float xs[4 * kRowBatch];
#pragma unroll
            for (int u = 0; u < 4 * kRowBatch; u++) {
                const int v = v0 + u * kTopkThreads;
                xs[u] = v < V ? __ldg(x + v) : 0.f;
            }
#pragma unroll
            for (int u = 0; u < 4 * kRowBatch; u++) {
                const int v = v0 + u * kTopkThreads;
                if (v < V) f(xs[u], v);
            }
        }
    }
}

// S blocks per (sequence, position) row, block j taking the slice
// [V j / S, V (j + 1) / S) of the row; keys key(x, v) order by (value desc,
// token asc).  Every block finds the exact top min(K, slice) keys of its
// slice; the global top K is among them.  Pass 1: every thread finds the
// largest key of its share of the slice.  Bound T: in every warp the m-th largest of these maxima
// (m = ceil(K/32), warp bitonic sort), minimised over the warps -- at least
// 32*m >= K threads hold a key >= T, so the K-th largest key is >= T, and
// only a small multiple of K keys reach it.  Pass 2 gathers the keys >= T
// (the slice is now in L2) and the top K of them are ranked in shared
// memory.  If more than kCollCap keys reach T (pathological rows, e.g. many
// equal values), an exact radix select over the slice decides instead: 12
// bits per pass from the top, the keys above the threshold digit taken, and
// once the threshold digit holds at most kCollCap keys they are gathered for
// an in-memory select.  With S > 1 each block publishes its keys (zeros past
// its count) and the last block of the row to finish (atomic ticket; nobody
// waits) selects the K largest of the S K published keys.
__global__ void __launch_bounds__(kTopkThreads)
    cand_topk_kernel(const float* dlog, int V, int K, int S, int* cand_tok, uint64_t* part, int* ticket,
                     int by_value, long long out_stride, float* out_val) {
    pdl_trigger();
    pdl_wait();
    extern __shared__ uint64_t csm[];
    uint64_t* coll = csm;                                       // [kCollCap]
    uint64_t* out = coll + kCollCap;                            // [K]
    uint64_t* surv = out + K;                                   // [kRankMax]
    uint32_t* hist = reinterpret_cast<uint32_t*>(surv + kRankMax);  // [kBins]
    __shared__ uint32_t hist8[256];
    __shared__ int scal[4];
    __shared__ uint64_t wmin[kTopkThreads / 32];
    __shared__ int dig[2];
    __shared__ int cnt[2];  // [0] keys taken into out, [1] keys gathered into coll
    __shared__ int last;
    const int row = blockIdx.x / S, sl = blockIdx.x % S;
    const int v0 = static_cast<int>(static_cast<long long>(V) * sl / S);
    const int Vs = static_cast<int>(static_cast<long long>(V) * (sl + 1) / S) - v0;
    const int Kl = min(K, Vs);  // keys this block selects from its slice
    const float* x = dlog + static_cast<size_t>(row) * V + v0;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (tid == 0) cnt[0] = cnt[1] = 0;
    // pass 1: this thread's largest key
    uint64_t mx = 0ull;
    for_row(x, Vs, [&](float xv, int v) {
        const uint64_t k = make_key(xv, static_cast<uint32_t>(v0 + v));
        mx = k > mx ? k : mx;
    });
    {
        const int m = (Kl + 31) / 32;
        uint64_t hv = mx;
#pragma unroll
        for (int size = 2; size <= 32; size <<= 1) {
#pragma unroll
            for (int stride = size >> 1; stride > 0; stride >>= 1) {
                const uint64_t y = shfl_xor_u64(hv, stride);
                const bool desc_block = (lane & size) == 0;
                const bool lower = (lane & stride) == 0;
                hv = (lower == desc_block) ? (hv > y ? hv : y) : (hv < y ? hv : y);
            }
        }
        const uint64_t mth = shfl_u64(hv, m - 1);
        if (lane == 0) wmin[warp] = mth;
    }
    __syncthreads();
    uint64_t T = wmin[0];
    for (int w = 1; w < kTopkThreads / 32; w++) T = wmin[w] < T ? wmin[w] : T;
    // pass 2: gather every key >= T
    for_row(x, Vs, [&](float xv, int v) {
        const uint64_t k = make_key(xv, static_cast<uint32_t>(v0 + v));
        if (k >= T) {
            const int pos = atomicAdd(&cnt[1], 1);
            if (pos < kCollCap) coll[pos] = k;
        }
    });
    __syncthreads();
    const int ng = cnt[1];
    const bool inexact = ng > kCollCap;
    __syncthreads();  // every thread has read the count before it is reused
    if (!inexact) {
        // the Kl largest of the ng gathered keys (ng >= Kl, keys distinct)
        if (ng <= kRankMax) {
            for (int i = tid; i < ng; i += kTopkThreads) {
                const uint64_t k = coll[i];
                int r = 0;
                for (int j = 0; j < ng; j++) r += coll[j] > k;
                if (r < Kl) out[r] = k;
            }
        } else {
            const uint64_t kth = block_kth_largest(coll, ng, Kl, hist8, scal);
            for (int i = tid; i < ng; i += kTopkThreads)
                if (coll[i] >= kth) out[atomicAdd(&cnt[0], 1)] = coll[i];
        }
        __syncthreads();
    }
    if (inexact) {
        if (tid == 0) cnt[0] = cnt[1] = 0;
        __syncthreads();
        uint64_t prefix = 0, mask = 0;
        int need = Kl;
        // at most 6 passes: after the 4-bit sixth digit the prefix is the whole
        // key, which is unique, so the threshold digit holds <= 1 key
        for (int level = 0, shift = 64 - kDigitBits; level < 6; level++, shift -= kDigitBits) {
            const int sh = shift > 0 ? shift : 0;
            const uint64_t dmask = (shift > 0 ? static_cast<uint64_t>(kBins - 1) : ((1ull << (kDigitBits + shift)) - 1));
            for (int i = tid; i < kBins; i += kTopkThreads) hist[i] = 0;
            __syncthreads();
            for (int v = tid; v < Vs; v += kTopkThreads) {
                const uint64_t k = make_key(__ldg(x + v), static_cast<uint32_t>(v0 + v));
                if ((k & mask) == prefix) atomicAdd(&hist[(k >> sh) & dmask], 1u);
            }
            __syncthreads();
            if (tid < 32) find_digit(hist, need, dig);
            __syncthreads();
            const uint64_t b = static_cast<uint64_t>(dig[0]);
            const int above = dig[1];
            const int m = static_cast<int>(hist[b]);
            const bool finish = m <= kCollCap;
            for (int v = tid; v < Vs; v += kTopkThreads) {
                const uint64_t k = make_key(__ldg(x + v), static_cast<uint32_t>(v0 + v));
                if ((k & mask) != prefix) continue;
                const uint64_t dg = (k >> sh) & dmask;
                if (dg > b)
                    out[atomicAdd(&cnt[0], 1)] = k;
                else if (dg == b && finish)
                    coll[atomicAdd(&cnt[1], 1)] = k;
            }
            __syncthreads();
            need -= above;
            if (finish) {
                // the `need` largest of the m gathered keys (keys are distinct)
                const uint64_t kth = need < m ? block_kth_largest(coll, m, need, hist8, scal) : 0ull;
                for (int i = tid; i < m; i += kTopkThreads)
                    if (coll[i] >= kth) out[atomicAdd(&cnt[0], 1)] = coll[i];
                __syncthreads();
                break;
            }
            prefix |= b << sh;
            mask |= dmask << sh;
            __syncthreads();
        }
    }
    if (S > 1) {
        // publish this slice's keys; the last block of the row merges
        uint64_t* pp = part + (static_cast<size_t>(row) * S + sl) * K;
        for (int i = tid; i < K; i += kTopkThreads) pp[i] = i < Kl ? out[i] : 0ull;
        __threadfence();
        __syncthreads();
        if (tid == 0) last = atomicAdd(&ticket[row], 1) == S - 1;
        __syncthreads();
        if (!last) return;
        __threadfence();
        if (tid == 0) {
            ticket[row] = 0;
            cnt[0] = 0;
        }
        // S K <= kCollCap keys, non-zero ones distinct, at least K of them
        const int ng = S * K;
        const uint64_t* rp = part + static_cast<size_t>(row) * S * K;
        for (int i = tid; i < ng; i += kTopkThreads) coll[i] = __ldcg(rp + i);
        __syncthreads();
        const uint64_t kth = block_kth_largest(coll, ng, K, hist8, scal);
        for (int i = tid; i < ng; i += kTopkThreads)
            if (coll[i] >= kth && coll[i] != 0ull) out[atomicAdd(&cnt[0], 1)] = coll[i];
        __syncthreads();
    }
    // write the K tokens in ascending token order, or (by_value) best first
    // with their values (rank by counting; keys are distinct)
    for (int i = tid; i < K; i += kTopkThreads) {
        const uint32_t tk = key_idx(out[i]);
        int r = 0;
        if (by_value) {
            for (int j = 0; j < K; j++) r += out[j] > out[i];
        } else {
            for (int j = 0; j < K; j++) r += key_idx(out[j]) < tk;
        }
        cand_tok[static_cast<size_t>(row) * out_stride + r] = static_cast<int>(tk);
        if (out_val) out_val[static_cast<size_t>(row) * out_stride + r] = key_val(out[i]);
    }
}

constexpr int kScoreWarps = 8;   // candidates per block (one per warp)
constexpr int kScoreThreads = kScoreWarps * 32;
constexpr int kScoreAcc = 8;     // node accumulators a lane keeps at once

// Block = (sequence s, group of kScoreWarps candidates, d-slice ds of DS):
// the block stages the slice of every node state of s in shared memory, warp
// w forms the partial dot products of candidate i = group*8 + w with them (a
// lane-strided partial sum in fixed order, then a butterfly) and writes them
// to scratch[ds][n][i].  The last block of (s, group) to finish (atomic
// ticket; nobody waits) sums the DS slices in order and writes the merge
// kernel's lists: deterministic.
__global__ void __launch_bounds__(kScoreThreads) cand_score_kernel(const CandArgs a) {
    pdl_trigger();
    pdl_wait();
    extern __shared__ float hs[];  // [P][dchunk]
    __shared__ int last;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int ngroups = (a.K + kScoreWarps - 1) / kScoreWarps;
    const int ds = blockIdx.x % a.DS;
    const int cg = (blockIdx.x / a.DS) % ngroups;
    const int s = blockIdx.x / (a.DS * ngroups);
    const int d = a.d, P = a.P, N = a.nseq * a.P;
    const int dchunk = d / a.DS, j0 = ds * dchunk, q = dchunk / 4;
    constexpr int kStageBatch = 4;  // loads in flight per thread while staging
    for (int u0 = tid; u0 < P * q; u0 += kStageBatch * kScoreThreads) {
        float4 v[kStageBatch];
#pragma unroll
        for (int b = 0; b < kStageBatch; b++) {
            const int u = u0 + b * kScoreThreads;
            if (u < P * q) {
                const int p = u / q, jj = (u % q) * 4;
                v[b] = *reinterpret_cast<const float4*>(a.h + static_cast<size_t>(s * P + p) * d + j0 + jj);
            }
        }
#pragma unroll
        for (int b = 0; b < kStageBatch; b++) {
            const int u = u0 + b * kScoreThreads;
            if (u < P * q) {
                const int p = u / q, jj = (u % q) * 4;
                *reinterpret_cast<float4*>(hs + p * dchunk + jj) = v[b];
            }
        }
    }
    __syncthreads();
    const size_t crow = (static_cast<size_t>(s) * a.L + a.dep - 1) * a.K;
    const int i = cg * kScoreWarps + warp;
    // a token outside the vocabulary would mean corrupted candidate lists:
    // it is never dereferenced (its score is -inf)
    if (i < a.K && static_cast<unsigned>(a.cand_tok[crow + i]) < static_cast<unsigned>(a.V)) {
        const int tok = a.cand_tok[crow + i];
        for (int p0 = 0; p0 < P; p0 += kScoreAcc) {
            float acc[kScoreAcc];
#pragma unroll
            for (int pp = 0; pp < kScoreAcc; pp++) acc[pp] = 0.0f;
            for (int j = lane * 4; j < dchunk; j += 128) {
                float4 ev;
                if (a.wbf16) {
                    const uint2 eb = __ldg(reinterpret_cast<const uint2*>(
                        static_cast<const __nv_bfloat16*>(a.E) + static_cast<size_t>(tok) * d + j0 + j));
                    const __nv_bfloat162 e01 = *reinterpret_cast<const __nv_bfloat162*>(&eb.x);
                    const __nv_bfloat162 e23 = *reinterpret_cast<const __nv_bfloat162*>(&eb.y);
                    ev = make_float4(__low2float(e01), __high2float(e01), __low2float(e23), __high2float(e23));
                } else {
                    ev = __ldg(reinterpret_cast<const float4*>(static_cast<const float*>(a.E) +
                                                               static_cast<size_t>(tok) * d + j0 + j));
                }
#pragma unroll
                for (int pp = 0; pp < kScoreAcc; pp++) {
                    if (p0 + pp < P) {
                        const float4 hv = *reinterpret_cast<const float4*>(hs + (p0 + pp) * dchunk + j);
                        float t = acc[pp];
                        t = fmaf(ev.x, hv.x, t);
                        t = fmaf(ev.y, hv.y, t);
                        t = fmaf(ev.z, hv.z, t);
                        acc[pp] = fmaf(ev.w, hv.w, t);
                    }
                }
            }
#pragma unroll
            for (int pp = 0; pp < kScoreAcc; pp++) {
                float v = acc[pp];
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
                if (lane == 0 && p0 + pp < P)
                    a.scratch[(static_cast<size_t>(ds) * N + s * P + p0 + pp) * a.K + i] = v;
            }
        }
    }
    __threadfence();
    __syncthreads();
    if (tid == 0) {
        const int tk = atomicAdd(&a.ticket[s * ngroups + cg], 1);
        last = tk == a.DS - 1;
        if (last) a.ticket[s * ngroups + cg] = 0;
    }
    __syncthreads();
    if (!last) return;
    __threadfence();
    const int stride = part_stride(a.K, 1);
    for (int u = tid; u < P * kScoreWarps; u += kScoreThreads) {
        const int p = u / kScoreWarps, ii = cg * kScoreWarps + u % kScoreWarps;
        if (ii >= a.K) continue;
        const int n = s * P + p;
        float dot = 0.0f;
        for (int r = 0; r < a.DS; r++) dot += __ldcg(a.scratch + (static_cast<size_t>(r) * N + n) * a.K + ii);
        const int tok = a.cand_tok[crow + ii];
        const bool ok = static_cast<unsigned>(tok) < static_cast<unsigned>(a.V);
        const float dl = ok ? a.dlog[static_cast<size_t>(s) * a.dlog_seq_stride + a.dlog_row_off + tok] : -INFINITY;
        float z = ok ? (dl + dot) * a.invT : -INFINITY;
        if (z == 0.0f) z = 0.0f;  // -0 -> +0
        a.part_ms[static_cast<size_t>(n) * a.K + ii] =
            z == -INFINITY ? make_float2(-INFINITY, 0.0f) : make_float2(z, 1.0f);
        a.part_key[static_cast<size_t>(n) * stride + ii] = make_key(z, static_cast<uint32_t>(tok));
    }
}

}  // namespace

int cand_topk_smem(int K) { return (kCollCap + K + kRankMax) * 8 + kBins * 4; }

// Blocks per row of the candidate top-K: slices of at least 4096 logits
// (several per thread of the block), at most 8, S K keys within the merge's
// shared-memory buffer, and rows x S within one block per SM (measured on
// GB300: 8 slices of 16 rows -2 % per round at K = 64; 8 slices of 128 rows,
// several waves, +2.4 %).
int cand_topk_slices(int V, int K, int rows, int num_sms) {
    const int s = std::min(std::min(8, V / 4096), std::min(kCollCap / K, num_sms / std::max(rows, 1)));
    return std::max(1, s);
}

int cand_score_slices(int P, int d, int nseq, int K, int max_smem) {
    // slices of d per block: enough blocks to spread the loads (>= 128), the
    // staged slice within 64 KB, and d / DS a multiple of 4 floats
    const int ngroups = (K + kScoreWarps - 1) / kScoreWarps;
    int DS = 1;
    while (d % (8 * DS) == 0 &&
           (static_cast<long long>(P) * (d / DS) * 4 > 64 * 1024 || nseq * ngroups * DS < 128))
        DS *= 2;
    if (static_cast<long long>(P) * (d / DS) * 4 > max_smem) return 0;
    return DS;
}

int cand_score_smem(int P, int d, int DS) { return P * (d / DS) * 4; }

cudaError_t cand_set_smem_limits() {
    cudaError_t e = set_max_dynamic_smem(reinterpret_cast<const void*>(cand_topk_kernel));
    if (e == cudaSuccess) e = set_max_dynamic_smem(reinterpret_cast<const void*>(cand_score_kernel));
    return e;
}

cudaError_t launch_cand_topk(const float* dlog, int rows, int V, int K, int S, int* cand_tok, uint64_t* part,
                             int* ticket, cudaStream_t st) {
    return launch_pdl(cand_topk_kernel, dim3(rows * S), dim3(kTopkThreads), cand_topk_smem(K), st, dlog, V, K, S,
                      cand_tok, part, ticket, 0, static_cast<long long>(K), static_cast<float*>(nullptr));
}

cudaError_t launch_row_topk_by_value(const float* x, int rows, int V, int K, int S, int* tok, float* val,
                                     long long out_stride, uint64_t* part, int* ticket, cudaStream_t st) {
    return launch_pdl(cand_topk_kernel, dim3(rows * S), dim3(kTopkThreads), cand_topk_smem(K), st, x, V, K, S, tok,
                      part, ticket, 1, out_stride, val);
}

cudaError_t launch_cand_score(const CandArgs& a, cudaStream_t st) {
    const int ngroups = (a.K + kScoreWarps - 1) / kScoreWarps;
    return launch_pdl(cand_score_kernel, dim3(a.nseq * ngroups * a.DS), dim3(kScoreThreads),
                      cand_score_smem(a.P, a.d, a.DS), st, a);
}

}  // namespace dart
