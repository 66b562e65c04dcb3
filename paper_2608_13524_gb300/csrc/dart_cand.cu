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
#include "dart_device.cuh"
#include "dart_kernels.h"

namespace dart {

namespace {

constexpr int kTopkThreads = 1024;
constexpr int kDigitBits = 12;
constexpr int kBins = 1 << kDigitBits;  // histogram bins per radix pass
constexpr int kCollCap = 4096;          // keys of the threshold bin finished in shared memory

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

// One block per (sequence, position) row.  Radix select on the 64-bit keys
// key(x, v) (value desc, token asc), 12 bits per pass from the top: a pass
// histograms the keys that match the prefix chosen so far, the keys above
// the threshold digit are taken, and as soon as the threshold digit holds at
// most kCollCap keys they are gathered to shared memory and the rest is an
// exact in-memory select.  Typical rows need two passes over the row.
__global__ void __launch_bounds__(kTopkThreads) cand_topk_kernel(const float* dlog, int V, int K, int* cand_tok) {
    pdl_trigger();
    pdl_wait();
    extern __shared__ uint64_t csm[];
    uint64_t* coll = csm;                                       // [kCollCap]
    uint64_t* out = coll + kCollCap;                            // [K]
    uint32_t* hist = reinterpret_cast<uint32_t*>(out + K);      // [kBins]
    __shared__ uint32_t hist8[256];
    __shared__ int scal[4];
    __shared__ int dig[2];
    __shared__ int cnt[2];  // [0] keys taken into out, [1] keys gathered into coll
    const float* x = dlog + static_cast<size_t>(blockIdx.x) * V;
    const int tid = threadIdx.x;
    if (tid == 0) cnt[0] = cnt[1] = 0;
    uint64_t prefix = 0, mask = 0;
    int need = K;
    // at most 6 passes: after the 4-bit sixth digit the prefix is the whole
    // key, which is unique, so the threshold digit holds <= 1 key
    for (int level = 0, shift = 64 - kDigitBits; level < 6; level++, shift -= kDigitBits) {
        const int sh = shift > 0 ? shift : 0;
        const uint64_t dmask = (shift > 0 ? static_cast<uint64_t>(kBins - 1) : ((1ull << (kDigitBits + shift)) - 1));
        for (int i = tid; i < kBins; i += kTopkThreads) hist[i] = 0;
        __syncthreads();
        for (int v = tid; v < V; v += kTopkThreads) {
            const uint64_t k = make_key(__ldg(x + v), static_cast<uint32_t>(v));
            if ((k & mask) == prefix) atomicAdd(&hist[(k >> sh) & dmask], 1u);
        }
        __syncthreads();
        if (tid < 32) find_digit(hist, need, dig);
        __syncthreads();
        const uint64_t b = static_cast<uint64_t>(dig[0]);
        const int above = dig[1];
        const int m = static_cast<int>(hist[b]);
        const bool finish = m <= kCollCap;
        for (int v = tid; v < V; v += kTopkThreads) {
            const uint64_t k = make_key(__ldg(x + v), static_cast<uint32_t>(v));
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
    // write the K tokens in ascending order (rank by counting)
    for (int i = tid; i < K; i += kTopkThreads) {
        const uint32_t t = key_idx(out[i]);
        int r = 0;
        for (int j = 0; j < K; j++) r += key_idx(out[j]) < t;
        cand_tok[static_cast<size_t>(blockIdx.x) * K + r] = static_cast<int>(t);
    }
}

constexpr int kScoreWarps = 8;  // candidates per block

// Block = (sequence s, kScoreWarps consecutive candidates); warp w scores
// candidate i = octet*8 + w against every node p < P of the sequence.  Each
// lane accumulates a strided partial dot product (fixed order), reduced by a
// butterfly: deterministic.
__global__ void __launch_bounds__(kScoreWarps * 32) cand_score_kernel(const CandArgs a) {
    pdl_trigger();
    pdl_wait();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int octets = (a.K + kScoreWarps - 1) / kScoreWarps;
    const int s = blockIdx.x / octets;
    const int i = (blockIdx.x % octets) * kScoreWarps + warp;
    if (i >= a.K) return;
    const int tok = a.cand_tok[(static_cast<size_t>(s) * a.L + a.dep - 1) * a.K + i];
    const float dl = a.dlog[static_cast<size_t>(s) * a.dlog_seq_stride + a.dlog_row_off + tok];
    const int d = a.d;
    const int stride = part_stride(a.K, 1);
    for (int p = 0; p < a.P; p++) {
        const int n = s * a.P + p;
        const float* h = a.h + static_cast<size_t>(n) * d;
        float acc = 0.0f;
        if (a.wbf16) {
            const __nv_bfloat16* e = static_cast<const __nv_bfloat16*>(a.E) + static_cast<size_t>(tok) * d;
            for (int j = lane * 4; j < d; j += 128) {
                const uint2 ev = __ldg(reinterpret_cast<const uint2*>(e + j));
                const float4 hv = *reinterpret_cast<const float4*>(h + j);
                const __nv_bfloat162 e01 = *reinterpret_cast<const __nv_bfloat162*>(&ev.x);
                const __nv_bfloat162 e23 = *reinterpret_cast<const __nv_bfloat162*>(&ev.y);
                acc = fmaf(__low2float(e01), hv.x, acc);
                acc = fmaf(__high2float(e01), hv.y, acc);
                acc = fmaf(__low2float(e23), hv.z, acc);
                acc = fmaf(__high2float(e23), hv.w, acc);
            }
        } else {
            const float* e = static_cast<const float*>(a.E) + static_cast<size_t>(tok) * d;
            for (int j = lane * 4; j < d; j += 128) {
                const float4 ev = __ldg(reinterpret_cast<const float4*>(e + j));
                const float4 hv = *reinterpret_cast<const float4*>(h + j);
                acc = fmaf(ev.x, hv.x, acc);
                acc = fmaf(ev.y, hv.y, acc);
                acc = fmaf(ev.z, hv.z, acc);
                acc = fmaf(ev.w, hv.w, acc);
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xFFFFFFFFu, acc, o);
        if (lane == 0) {
            float z = (dl + acc) * a.invT;
            if (z == 0.0f) z = 0.0f;  // -0 -> +0
            a.part_ms[static_cast<size_t>(n) * a.K + i] = z == -INFINITY ? make_float2(-INFINITY, 0.0f)
                                                                        : make_float2(z, 1.0f);
            a.part_key[static_cast<size_t>(n) * stride + i] = make_key(z, static_cast<uint32_t>(tok));
        }
    }
}

}  // namespace

int cand_topk_smem(int K) { return (kCollCap + K) * 8 + kBins * 4; }

cudaError_t cand_set_smem_limits(int max_dyn) {
    return cudaFuncSetAttribute(cand_topk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, max_dyn);
}

cudaError_t launch_cand_topk(const float* dlog, int rows, int V, int K, int* cand_tok, cudaStream_t st) {
    return launch_pdl(cand_topk_kernel, dim3(rows), dim3(kTopkThreads), cand_topk_smem(K), st, dlog, V, K, cand_tok);
}

cudaError_t launch_cand_score(const CandArgs& a, cudaStream_t st) {
    const int octets = (a.K + kScoreWarps - 1) / kScoreWarps;
    return launch_pdl(cand_score_kernel, dim3(a.nseq * octets), dim3(kScoreWarps * 32), 0, st, a);
}

}  // namespace dart
