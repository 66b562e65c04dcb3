// The whole DARTree round of a small fp32 problem in one cooperative kernel.
//
// Small problems (fp32 weights, at most 32 nodes per depth, d <= 1024,
// V <= 65536) are latency-bound: at one launch per step the round is a chain
// of a dozen launches, each a few microseconds of launch and dependency
// latency around well under a microsecond of arithmetic.  Here every block
// of one grid (one block per SM, all resident: a cooperative launch) runs
// every step of every depth, with a grid-wide barrier where a step needs the
// whole result of the previous one:
//
//   A  scoring (Algorithm 1: every prefix of S_{d-1} over the full
//      vocabulary): block b takes a slice of vocabulary rows, stages the
//      normalised node states, forms z[n][v] = (Dlog[seq][d-1][v] +
//      E[v] . h[n]) / T and writes per node its (max, sum exp) and its k best
//      keys of the slice;
//   B  merge + "retain the global top-W" (one block per sequence): per node
//      the log-sum-exp over the slices and the k best of the slices' lists,
//      log q~ = min(z - lse, 0); then the frontier by Eq. 5 (the same
//      selection code as the multi-launch path) and, after depth L, prune and
//      emit (Lemma 1; also the multi-launch path's code);
//   C1 first head layer: a_c = SiLU(W_i [h_p ; E[t_c]]), a warp per output
//      feature over all children;
//   C2 second layer and residual: r_c = h_p + W_o a_c, with per-block sums
//      of r_c^2; the next depth's A normalises, h_c = r_c / rms(r_c).
//
// Sums run in a fixed order (lane-strided chunks, then a butterfly, then the
// blocks in index order), so the result is deterministic.  The grid barrier
// waits with the same 2 s limit as every other wait: a block that gives up
// sets the timeout bit of the status word and the abort flag, and every
// block returns at its next barrier.
#include "dart_device.cuh"
#include "dart_emit.cuh"
#include "dart_frontier.cuh"
#include "dart_kernels.h"

namespace dart {

namespace {

constexpr int kRoundThreads = 256;
constexpr int kRoundWarps = kRoundThreads / 32;

__device__ __forceinline__ unsigned ld_acquire_u32(const unsigned* p) {
    unsigned v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// Sense-reversing grid barrier over `nblocks` resident blocks.  bar[0]
// counts arrivals and bar[32] is the generation (another 128-byte line, so
// the polling does not meet the arrivals' atomics).  The last block to
// arrive resets the count and publishes the next generation; the others poll
// for it with the time limit (and leave early once any block has aborted).
// Returns false after a timeout or an abort: the caller returns.
__device__ bool grid_barrier(unsigned* bar, unsigned nblocks, int* abort, int* status, int* sflag,
                             unsigned long long limit_ns = kWaitLimitNs) {
    __syncthreads();
    if (threadIdx.x == 0) {
        int ok = 1;
        unsigned* gen_p = bar + 32;
        const unsigned gen = ld_acquire_u32(gen_p);
        // the release orders this block's writes (every thread's: they
        // happen before it through the block barrier above) before the arrival
        unsigned arrived;
        asm volatile("atom.add.release.gpu.global.u32 %0, [%1], 1;" : "=r"(arrived) : "l"(bar) : "memory");
        if (arrived == nblocks - 1) {
            asm volatile("st.relaxed.gpu.global.u32 [%0], 0;" ::"l"(bar) : "memory");
            asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(gen_p), "r"(gen + 1u) : "memory");
        } else {
            const unsigned long long t0 = globaltimer_ns();
            for (unsigned it = 1;; it++) {
                if (ld_acquire_u32(gen_p) != gen) break;
                if ((it & 63u) == 0u) {
                    if (*reinterpret_cast<volatile int*>(abort) != 0) {
                        ok = 0;
                        break;
                    }
                    if (globaltimer_ns() - t0 > limit_ns) {
                        atomicExch(abort, 1);
                        atomicOr(status, kDevTimeout);
                        ok = 0;
                        break;
                    }
                }
            }
        }
        *sflag = ok;
    }
    __syncthreads();
    return *sflag != 0;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
    return v;
}

__device__ __forceinline__ uint64_t warp_max_key(uint64_t v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const uint64_t w = __shfl_xor_sync(kFull, v, o);
        v = w > v ? w : v;
    }
    return v;
}

// Block b's vocabulary slice [v0, v1) of the V rows (balanced split).
__device__ __forceinline__ int slice_begin(const RoundArgs& a, int b) {
    return static_cast<int>((static_cast<long long>(b) * a.V) / a.G);
}

// Row pitch (floats) of the block's cached E slice: d + 4 keeps the float4
// reads of 32 consecutive rows (one per lane) on distinct bank groups.
__device__ __forceinline__ int es_pitch(int d) { return d + 4; }

// A: scores of block b's vocabulary slice for the N nodes of depth dep:
// z[n][v] = (Dlog[seq(n)][dep-1][v] + E[v] . h[n]) / T as selection keys,
// then per node its (max, sum exp) and its k best keys, in order.
template <int NM>
__device__ void score_slice(const RoundArgs& a, int dep, int N, int P, const float* es, float* hs, float* red,
                            uint64_t* kz) {
    const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
    const int d = a.d, d4 = d / 4;
    const int v0 = slice_begin(a, b), R = slice_begin(a, b + 1) - v0;
    float* hcur = (dep & 1) ? a.h0 : a.h1;  // depth dep's states (parity buffer)
    // stage the normalised states (the raw rows and the sums of squares are
    // requested together); block n % G also writes state n out
    for (int n = w; n < N; n += kRoundWarps) {
        const float4* src = reinterpret_cast<const float4*>(dep == 1 ? a.anchor + static_cast<size_t>(n / P) * d
                                                                    : a.rbuf + static_cast<size_t>(n) * d);
        constexpr int kQ = 8;  // d <= 1024: at most 8 float4 per lane
        float4 x[kQ];
#pragma unroll
        for (int u = 0; u < kQ; u++) {
            const int q = lane + 32 * u;
            if (q < d4) x[u] = dep == 1 ? __ldg(src + q) : __ldcg(src + q);
        }
        float sc = 1.0f;
        if (dep > 1) {
            constexpr int kB = 5;  // G <= 160
            float part[kB];
#pragma unroll
            for (int u = 0; u < kB; u++) {
                const int bb = lane + 32 * u;
                part[u] = bb < a.G ? __ldcg(a.ssqp + static_cast<size_t>(n) * a.G + bb) : 0.0f;
            }
            float t = 0.0f;
#pragma unroll
            for (int u = 0; u < kB; u++) t += part[u];
            t = warp_sum(t);
            sc = rsqrtf(t / static_cast<float>(d) + a.eps);
        }
        float4* dst = reinterpret_cast<float4*>(hs + static_cast<size_t>(n) * d);
        float4* out = reinterpret_cast<float4*>(hcur + static_cast<size_t>(n) * d);
#pragma unroll
        for (int u = 0; u < kQ; u++) {
            const int q = lane + 32 * u;
            if (q < d4) {
                float4 y = x[u];
                y.x *= sc;
                y.y *= sc;
                y.z *= sc;
                y.w *= sc;
                dst[q] = y;
                if (n % a.G == b) out[q] = y;
            }
        }
    }
    __syncthreads();
    const float4* hs4 = reinterpret_cast<const float4*>(hs);
    const float4* E4 = reinterpret_cast<const float4*>(a.E);
    const int ep4 = es_pitch(d) / 4;
    const int q0 = w * (d4 / kRoundWarps), q1 = (w + 1) * (d4 / kRoundWarps);
    const size_t drow = static_cast<size_t>(dep - 1) * a.V;
    for (int r0 = 0; r0 < R; r0 += 32) {
        const int r = r0 + lane;
        const bool valid = r < R;
        float acc[NM];
#pragma unroll
        for (int n = 0; n < NM; n++) acc[n] = 0.0f;
        if (valid) {
            const float4* er = es ? reinterpret_cast<const float4*>(es) + static_cast<size_t>(r) * ep4
                                  : E4 + static_cast<size_t>(v0 + r) * d4;
            for (int q = q0; q < q1; q++) {
                const float4 e = es ? er[q] : __ldg(er + q);
#pragma unroll
                for (int n = 0; n < NM; n++) {
                    if (n < N) {
                        const float4 h = hs4[n * d4 + q];
                        acc[n] = fmaf(e.x, h.x, acc[n]);
                        acc[n] = fmaf(e.y, h.y, acc[n]);
                        acc[n] = fmaf(e.z, h.z, acc[n]);
                        acc[n] = fmaf(e.w, h.w, acc[n]);
                    }
                }
            }
        }
#pragma unroll
        for (int n = 0; n < NM; n++)
            if (n < N) red[(w * NM + n) * 32 + lane] = acc[n];
        __syncthreads();
        for (int t = tid; t < N * 32; t += kRoundThreads) {
            const int n = t >> 5, l = t & 31;
            if (r0 + l < R) {
                float sdot = 0.0f;
#pragma unroll
                for (int ww = 0; ww < kRoundWarps; ww++) sdot += red[(ww * NM + n) * 32 + l];
                const int vv = v0 + r0 + l;
                const float dl = __ldg(a.dlog + static_cast<size_t>(n / P) * a.L * a.V + drow + vv);
                kz[n * a.R + r0 + l] = make_key((sdot + dl) * a.invT, static_cast<uint32_t>(vv));
            }
        }
        __syncthreads();
    }
    for (int n = w; n < N; n += kRoundWarps) {
        uint64_t* kn = kz + n * a.R;
        float m = -INFINITY;
        for (int i = lane; i < R; i += 32) m = fmaxf(m, key_val(kn[i]));
        m = warp_max(m);
        float s = 0.0f;
        if (m != -INFINITY)
            for (int i = lane; i < R; i += 32) {
                const float z = key_val(kn[i]);
                if (z != -INFINITY) s += __expf(z - m);
            }
        s = warp_sum(s);
        if (lane == 0) a.pms[static_cast<size_t>(n) * a.G + b] = make_float2(m, s);
        uint64_t* out = a.pkey + (static_cast<size_t>(n) * a.G + b) * a.k;
        for (int j = 0; j < a.k; j++) {
            uint64_t best = 0ull;
            int at = -1;
            for (int i = lane; i < R; i += 32)
                if (kn[i] > best) {
                    best = kn[i];
                    at = i;
                }
            const uint64_t top = warp_max_key(best);
            if (top != 0ull && best == top) kn[at] = 0ull;  // keys are distinct: one owner
            if (lane == 0) out[j] = top;
            __syncwarp();
        }
    }
}

// B, per node of sequence s: log-sum-exp and the k best keys over the G
// slices, written as the node's sorted children (warp w, nodes p = w, w+8..).
// With `stage` (G * k keys per warp of shared memory) a node's lists are
// read in one batch of loads and merged from shared memory.
__device__ void merge_nodes(const RoundArgs& a, int s, int P, int prev_count, uint64_t* stage) {
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    constexpr int kLists = 5;  // G <= 160 slices: lane l owns slices l + 32 i
    const int gk = a.G * a.k;
    uint64_t* mine = stage ? stage + static_cast<size_t>(w) * gk : nullptr;
    for (int p = w; p < P; p += kRoundWarps) {
        const int n = s * P + p;
        float* lq_out = a.node_logq + static_cast<size_t>(n) * a.k;
        int* tok_out = a.node_tok + static_cast<size_t>(n) * a.k;
        if (p >= prev_count) {
            for (int j = lane; j < a.k; j += 32) {
                lq_out[j] = -INFINITY;
                tok_out[j] = -1;
            }
            if (lane == 0) a.node_lse[n] = -INFINITY;
            continue;
        }
        const uint64_t* lists = a.pkey + static_cast<size_t>(n) * gk;
        if (mine) {
            // eight loads in flight per lane before their stores
            for (int i0 = 0; i0 < gk; i0 += 256) {
                uint64_t v[8];
#pragma unroll
                for (int u = 0; u < 8; u++) {
                    const int i = i0 + lane + 32 * u;
                    v[u] = i < gk ? __ldcg(lists + i) : 0ull;
                }
#pragma unroll
                for (int u = 0; u < 8; u++) {
                    const int i = i0 + lane + 32 * u;
                    if (i < gk) mine[i] = v[u];
                }
            }
        }
        float2 pm[kLists];
#pragma unroll
        for (int u = 0; u < kLists; u++) {
            const int bb = lane + 32 * u;
            pm[u] = bb < a.G ? __ldcg(a.pms + static_cast<size_t>(n) * a.G + bb) : make_float2(-INFINITY, 0.0f);
        }
        float2 acc = make_float2(-INFINITY, 0.0f);
#pragma unroll
        for (int u = 0; u < kLists; u++) acc = lse_merge(acc, pm[u]);
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            float2 other;
            other.x = __shfl_xor_sync(kFull, acc.x, o);
            other.y = __shfl_xor_sync(kFull, acc.y, o);
            // the lower lane's partial first: both lanes form the same sum
            acc = (lane & o) ? lse_merge(other, acc) : lse_merge(acc, other);
        }
        const float lse = acc.x == -INFINITY ? -INFINITY : acc.x + logf(acc.y);
        __syncwarp();
        const uint64_t* src = mine ? mine : lists;
        int ptr[kLists];
        uint64_t head[kLists];
#pragma unroll
        for (int i = 0; i < kLists; i++) {
            const int l = lane + 32 * i;
            ptr[i] = 0;
            head[i] = l < a.G ? (mine ? src[l * a.k] : __ldcg(src + static_cast<size_t>(l) * a.k)) : 0ull;
        }
        for (int j = 0; j < a.k; j++) {
            uint64_t best = 0ull;
#pragma unroll
            for (int i = 0; i < kLists; i++) best = head[i] > best ? head[i] : best;
            const uint64_t top = warp_max_key(best);
#pragma unroll
            for (int i = 0; i < kLists; i++) {
                if (top != 0ull && head[i] == top) {
                    const int l = lane + 32 * i;
                    ptr[i]++;
                    const size_t at = static_cast<size_t>(l) * a.k + ptr[i];
                    head[i] = ptr[i] < a.k ? (mine ? src[at] : __ldcg(src + at)) : 0ull;
                }
            }
            if (lane == 0) {
                const float z = top != 0ull ? key_val(top) : -INFINITY;
                lq_out[j] = (lse != -INFINITY && z != -INFINITY) ? fminf(z - lse, 0.0f) : -INFINITY;
                tok_out[j] = top != 0ull ? static_cast<int>(key_idx(top)) : -1;
            }
        }
        if (lane == 0) a.node_lse[n] = lse;
        __syncwarp();
    }
}

// sum over the n4 float4 of w . x, lane-strided then a butterfly (fixed
// order); up to 8 float4 per lane requested at once.  Every lane returns it.
__device__ __forceinline__ float warp_dot(const float4* w, const float4* x, int n4, bool x_l2, int lane) {
    float acc = 0.0f;
    for (int q0 = 0; q0 < n4; q0 += 256) {
        float4 wv[8], xv[8];
#pragma unroll
        for (int u = 0; u < 8; u++) {
            const int q = q0 + lane + 32 * u;
            if (q < n4) {
                wv[u] = __ldg(w + q);
                xv[u] = x_l2 ? __ldcg(x + q) : __ldg(x + q);
            }
        }
#pragma unroll
        for (int u = 0; u < 8; u++) {
            if (q0 + lane + 32 * u < n4) {
                acc = fmaf(wv[u].x, xv[u].x, acc);
                acc = fmaf(wv[u].y, xv[u].y, acc);
                acc = fmaf(wv[u].z, xv[u].z, acc);
                acc = fmaf(wv[u].w, xv[u].w, acc);
            }
        }
    }
    return warp_sum(acc);
}

// C1: a[c][i] = SiLU(W_i[i] . [h_p ; E[t_c]]) for the Nc child slots (zero
// for an empty slot; Np parent rows): one warp per (feature, child) task.
__device__ void head_layer1(const RoundArgs& a, int dep, int Np, int Nc) {
    const int lane = threadIdx.x & 31;
    const int gw = blockIdx.x * kRoundWarps + (threadIdx.x >> 5), tw = a.G * kRoundWarps;
    const int d = a.d, d4 = d / 4;
    const float* hcur = (dep & 1) ? a.h0 : a.h1;
    for (int t = gw; t < d * Nc; t += tw) {
        const int i = t / Nc, c = t % Nc;
        const int pr = __ldcg(a.child_prow + c), tk = __ldcg(a.child_tok + c);
        const bool tok_ok = static_cast<unsigned>(tk) < static_cast<unsigned>(a.V);
        (void)bounds_check(a.status, pr < 0 || (tok_ok && pr < Np));
        float u = 0.0f;
        if (pr >= 0 && tok_ok) {
            const float4* wr = reinterpret_cast<const float4*>(a.Wi + static_cast<size_t>(i) * 2 * d);
            u = warp_dot(wr, reinterpret_cast<const float4*>(hcur + static_cast<size_t>(pr) * d), d4, true, lane) +
                warp_dot(wr + d4, reinterpret_cast<const float4*>(a.E + static_cast<size_t>(tk) * d), d4, false, lane);
            u = u / (1.0f + __expf(-u));
        }
        if (lane == 0) a.abuf[static_cast<size_t>(c) * d + i] = u;
    }
}

// C2: r[c][i] = h_p[i] + W_o[i] . a_c (zero for an empty slot), and this
// block's sum of r[c][i]^2 over its tasks, per child (warps in order).
__device__ void head_layer2(const RoundArgs& a, int dep, int Nc, float* sq) {
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    const int gw = blockIdx.x * kRoundWarps + w, tw = a.G * kRoundWarps;
    const int d = a.d, d4 = d / 4;
    const float* hcur = (dep & 1) ? a.h0 : a.h1;
    for (int c = lane; c < Nc; c += 32) sq[w * 32 + c] = 0.0f;
    __syncwarp();
    for (int t = gw; t < d * Nc; t += tw) {
        const int i = t / Nc, c = t % Nc;
        const int pr = __ldcg(a.child_prow + c);
        float r = 0.0f;
        if (pr >= 0) {
            const float hp = __ldcg(hcur + static_cast<size_t>(pr) * d + i);
            const float y = warp_dot(reinterpret_cast<const float4*>(a.Wo + static_cast<size_t>(i) * d),
                                     reinterpret_cast<const float4*>(a.abuf + static_cast<size_t>(c) * d), d4, true,
                                     lane);
            r = hp + y;
        }
        if (lane == 0) {
            a.rbuf[static_cast<size_t>(c) * d + i] = r;
            sq[w * 32 + c] = fmaf(r, r, sq[w * 32 + c]);
        }
    }
    __syncthreads();
    for (int c = threadIdx.x; c < Nc; c += kRoundThreads) {
        float t = 0.0f;
        for (int ww = 0; ww < kRoundWarps; ww++) t += sq[ww * 32 + c];
        a.ssqp[static_cast<size_t>(c) * a.G + blockIdx.x] = t;
    }
}

// B for sequence s at depth dep (merge, frontier, and after depth L prune
// and emit), by the calling block.
__device__ void select_sequence(const RoundArgs& a, SelectArgs& sa, int dep, int s, int N, int P, int Pn,
                                uint64_t* keys, int* ctok, uint64_t* surv, uint64_t* top, uint64_t* stage,
                                uint64_t* thr, uint32_t* hist, int* scal, int* redi) {
    const int prev_count = dep == 1 ? 1 : __ldcg(a.tree_count + s * a.L + dep - 2);
    merge_nodes(a, s, P, prev_count, stage);
    __syncthreads();
    sa.N = N;
    sa.P = P;
    sa.dep = dep;
    sa.Pn = Pn;
    select_frontier(sa, s, prev_count, keys, ctok, surv, top, thr, hist, scal, redi);
    if (dep == a.L) {
        __syncthreads();
        prune_emit_seq<kRoundThreads>(a.emit, s);
    }
    __syncthreads();
}

template <int NM>
__global__ void __launch_bounds__(kRoundThreads, 1) round_small_f32_kernel(const RoundArgs a) {
    extern __shared__ __align__(16) uint8_t rsm[];
    __shared__ uint64_t thr;
    __shared__ uint32_t hist[256];
    __shared__ int scal[4];
    __shared__ int redi[32];
    __shared__ float sq[kRoundWarps * 32];
    __shared__ int sflag;
    // [the block's E slice, kept for the whole round (ecache)], then
    // A: states [NM][d], warp partials [8][NM][32], slice keys [NM][R];
    // B (aliases A): candidate keys [W*k], survivors, top 64, tokens [W*k],
    //    per-warp list staging [8][G*k] (mstage)
    const int d = a.d;
    const int R = slice_begin(a, blockIdx.x + 1) - slice_begin(a, blockIdx.x);
    float* es = a.ecache ? reinterpret_cast<float*>(rsm) : nullptr;
    uint8_t* un = rsm + (a.ecache ? static_cast<size_t>(a.R) * es_pitch(d) * 4 : 0);
    float* hs = reinterpret_cast<float*>(un);
    float* red = hs + NM * d;
    uint64_t* kz = reinterpret_cast<uint64_t*>(red + kRoundWarps * NM * 32);
    uint64_t* keys = reinterpret_cast<uint64_t*>(un);
    uint64_t* surv = keys + a.W * a.k;
    uint64_t* top = surv + kRankMax;
    uint64_t* stage = a.mstage ? top + 64 : nullptr;
    int* ctok = reinterpret_cast<int*>(top + 64 + (a.mstage ? kRoundWarps * a.G * a.k : 0));
    const unsigned G = static_cast<unsigned>(a.G);

    if (es) {
        // the slice of E this block scores at every depth
        const int v0 = slice_begin(a, blockIdx.x), d4 = d / 4, ep4 = es_pitch(d) / 4;
        const float4* E4 = reinterpret_cast<const float4*>(a.E);
        for (int q0 = 0; q0 < R * d4; q0 += 8 * kRoundThreads) {
            float4 v[8];  // eight loads in flight per thread before their stores
#pragma unroll
            for (int u = 0; u < 8; u++) {
                const int q = q0 + threadIdx.x + u * kRoundThreads;
                if (q < R * d4) v[u] = __ldg(E4 + static_cast<size_t>(v0) * d4 + q);
            }
#pragma unroll
            for (int u = 0; u < 8; u++) {
                const int q = q0 + threadIdx.x + u * kRoundThreads;
                if (q < R * d4) reinterpret_cast<float4*>(es)[(q / d4) * ep4 + q % d4] = v[u];
            }
        }
        __syncthreads();
    }

    SelectArgs sa;
    sa.k = a.k;
    sa.W = a.W;
    sa.L = a.L;
    sa.nseq = a.nseq;
    sa.beta = a.beta;
    sa.node_logq = a.node_logq;
    sa.node_tok = a.node_tok;
    sa.node_lse = a.node_lse;
    sa.tree_tok = a.tree_tok;
    sa.tree_parent = a.tree_parent;
    sa.tree_score = a.tree_score;
    sa.tree_count = a.tree_count;
    sa.child_prow = a.child_prow;
    sa.child_tok = a.child_tok;
    sa.status = a.status;

    for (int dep = 1; dep <= a.L; dep++) {
        const int P = a.caps[dep - 1], Pn = a.caps[dep];
        const int N = a.nseq * P;
        score_slice<NM>(a, dep, N, P, es, hs, red, kz);
        if (a.nseq == 1) {
            // one sequence: the last block to finish its slice merges and
            // selects (an arrival ticket: nobody waits for it here)
            __syncthreads();
            if (threadIdx.x == 0) {
                int last;
                asm volatile("atom.add.acq_rel.gpu.global.u32 %0, [%1], 1;" : "=r"(last) : "l"(a.bar + 64) : "memory");
                sflag = static_cast<unsigned>(last) == G - 1u;
            }
            __syncthreads();
            if (sflag) {
                select_sequence(a, sa, dep, 0, N, P, Pn, keys, ctok, surv, top, stage, &thr, hist, scal, redi);
                if (threadIdx.x == 0) atomicExch(a.bar + 64, 0u);
            }
        } else {
            if (!grid_barrier(a.bar, G, a.abort, a.status, &sflag)) return;
            for (int s = blockIdx.x; s < a.nseq; s += a.G)
                select_sequence(a, sa, dep, s, N, P, Pn, keys, ctok, surv, top, stage, &thr, hist, scal, redi);
        }
        if (dep == a.L) break;
        if (!grid_barrier(a.bar, G, a.abort, a.status, &sflag)) return;
        head_layer1(a, dep, N, a.nseq * Pn);
        if (!grid_barrier(a.bar, G, a.abort, a.status, &sflag)) return;
        head_layer2(a, dep, a.nseq * Pn, sq);
        if (!grid_barrier(a.bar, G, a.abort, a.status, &sflag)) return;
    }
}

// ------------------------------------------------------------------------
// One thread-block cluster per sequence (kCS blocks): the same steps with
// the cluster's hardware barrier (a fraction of a microsecond, against about
// two for a grid-wide barrier) and the per-block partial results exchanged
// through distributed shared memory instead of global memory.  Sequences are
// independent, so the clusters never wait on one another.  Block r of the
// cluster scores vocabulary rows [r V / kCS, (r+1) V / kCS) and owns head
// features [r F, (r+1) F), F = d / kCS; every block keeps the depth's node
// states of its sequence in shared memory.

constexpr int kCS = kRoundCluster;

__device__ __forceinline__ uint32_t cl_addr(const void* local, uint32_t rank) {
    uint32_t remote;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(local)), "r"(rank));
    return remote;
}
__device__ __forceinline__ uint64_t ld_cl_u64(const void* local, uint32_t rank) {
    uint64_t v;
    asm volatile("ld.shared::cluster.u64 %0, [%1];" : "=l"(v) : "r"(cl_addr(local, rank)) : "memory");
    return v;
}
__device__ __forceinline__ float2 ld_cl_f32x2(const void* local, uint32_t rank) {
    float2 v;
    asm volatile("ld.shared::cluster.v2.f32 {%0, %1}, [%2];" : "=f"(v.x), "=f"(v.y) : "r"(cl_addr(local, rank)) : "memory");
    return v;
}
__device__ __forceinline__ uint32_t ld_cl_u32(const void* local, uint32_t rank) {
    uint32_t v;
    asm volatile("ld.shared::cluster.u32 %0, [%1];" : "=r"(v) : "r"(cl_addr(local, rank)) : "memory");
    return v;
}
__device__ __forceinline__ float ld_cl_f32(const void* local, uint32_t rank) {
    float v;
    asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(cl_addr(local, rank)) : "memory");
    return v;
}

__device__ __forceinline__ float dot4(const float4 a, const float4 b, float acc) {
    acc = fmaf(a.x, b.x, acc);
    acc = fmaf(a.y, b.y, acc);
    acc = fmaf(a.z, b.z, acc);
    return fmaf(a.w, b.w, acc);
}

// Candidates per lane of the warp-level frontier selection (at most
// 32 * kCandLane = W * k candidates).
constexpr int kCandLane = 8;

// The frontier of the cluster's sequence s by warp 0 of rank 0: the same keys
// and order as select_frontier (score desc, then candidate p * k + j asc).
// The children's lists come from the shared memory of the blocks that merged
// them (node p: block p % kCS, nlq / ntok [p][k]); the previous frontier's
// scores, the children (local parent slot, token) and the count stay in rank
// 0's shared memory for the next steps, and the supertree row, the child
// slots and the count also go to global memory (test hooks, prune / emit).
__device__ void select_frontier_cluster(const SelectArgs& a, int s, int prev_count, const float* nlq,
                                        const int* ntok, float* fscore, int* cprow, int* ctokr, int* fcount) {
    const int lane = threadIdx.x & 31;
    const int ncand = prev_count * a.k;
    uint64_t key[kCandLane];
    int tok[kCandLane];
    int valid = 0;
#pragma unroll
    for (int u = 0; u < kCandLane; u++) {
        const int c = lane + 32 * u;
        key[u] = 0ull;
        tok[u] = -1;
        if (c < ncand) {
            const int pp = c / a.k;
            const uint32_t owner = static_cast<uint32_t>(pp % kCS);
            const float ps = a.dep == 1 ? 0.0f : fscore[pp];
            const float sc = (ps + ld_cl_f32(nlq + c, owner)) + a.beta;  // Eq. 5, one more depth
            tok[u] = static_cast<int>(ld_cl_u32(ntok + c, owner));
            if (sc > -INFINITY) {
                key[u] = make_key(sc, static_cast<uint32_t>(c));
                valid++;
            }
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) valid += __shfl_xor_sync(kFull, valid, o);
    const int cnt = min(a.W, valid);
    __syncwarp();  // every lane has read fscore before it is overwritten
    const size_t tb = (static_cast<size_t>(s) * a.L + a.dep - 1) * a.W;
    auto keep = [&](int r, uint64_t tp, int tk) {
        const int pp = static_cast<int>(key_idx(tp)) / a.k;
        const float sc = key_val(tp);
        fscore[r] = sc;
        a.tree_tok[tb + r] = tk;
        a.tree_parent[tb + r] = a.dep == 1 ? -1 : pp;
        a.tree_score[tb + r] = sc;
        if (r < a.Pn) {
            cprow[r] = pp;
            ctokr[r] = tk;
            a.child_prow[s * a.Pn + r] = s * a.P + pp;
            a.child_tok[s * a.Pn + r] = tk;
        }
    };
    auto empty = [&](int r) {
        a.tree_tok[tb + r] = -1;
        a.tree_parent[tb + r] = -1;
        a.tree_score[tb + r] = -INFINITY;
        if (r < a.Pn) {
            cprow[r] = -1;
            ctokr[r] = 0;
            a.child_prow[s * a.Pn + r] = -1;
            a.child_tok[s * a.Pn + r] = 0;
        }
    };
    if (ncand <= 32) {
        // one candidate per lane: its rank among all keys (distinct) in one
        // pass of 32 independent shuffles instead of W dependent maxima
        const uint64_t mine = key[0];
        int rank = 0;
#pragma unroll
        for (int src = 0; src < 32; src++) rank += shfl_u64(mine, src) > mine ? 1 : 0;
        if (mine != 0ull && rank < cnt) keep(rank, mine, tok[0]);
        for (int r = cnt + lane; r < a.W; r += 32) empty(r);
        if (lane == 0) {
            *fcount = cnt;
            a.tree_count[s * a.L + a.dep - 1] = cnt;
        }
        return;
    }
    for (int r = 0; r < a.W; r++) {
        uint64_t best = 0ull;
#pragma unroll
        for (int u = 0; u < kCandLane; u++) best = key[u] > best ? key[u] : best;
        const uint64_t tp = warp_max_key(best);  // nonzero for r < cnt
        if (r < cnt) {
#pragma unroll
            for (int u = 0; u < kCandLane; u++) {
                if (key[u] == tp) {  // the one owner lane (the keys are distinct)
                    key[u] = 0ull;
                    keep(r, tp, tok[u]);
                }
            }
        } else if (lane == 0) {
            empty(r);
        }
    }
    if (lane == 0) {
        *fcount = cnt;
        a.tree_count[s * a.L + a.dep - 1] = cnt;
    }
}

template <int NP>
__global__ void __launch_bounds__(kRoundThreads, 1) round_cluster_f32_kernel(const RoundArgs a) {
    extern __shared__ __align__(16) uint8_t csm[];
    __shared__ float2 pms_s[32];  // this block's (max, sum exp) per node
    __shared__ float ssq_s[32];   // this block's sum of r^2 over its features, per child
    __shared__ __align__(8) uint64_t sbar[3];  // E stages 0, 1; [2] the resident head weights
    __shared__ int misc[2];       // [0] abort flag of this block
    __shared__ int cpar[32];      // C1 / C2: each child's parent slot (-1: empty or invalid)
    __shared__ int cpar_tok[32];  // and its token
    __shared__ float fscore[32];  // rank 0: the current frontier's scores
    __shared__ int cprow[32], ctokr[32];  // rank 0: the children (parent slot, token)
    __shared__ int fcount;        // rank 0: the current frontier's size
    constexpr int RS = 32 / NP;   // rows per warp step of the scoring
    const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
    const int s = blockIdx.x / kCS;
    const uint32_t rank = cluster_ctarank();
    const int d = a.d, d4 = d / 4, F = d / kCS, k = a.k;
    // states [NP][d] | slice keys [NP][k] | a slice, r slice, r^2 [NP][F] |
    // E stages [2][stage_bytes] | slice keys [NP][R] | children's E rows
    // [NP][d] (C1) / gathered a [NP][d] (C2) | merged lists [NP][k] x 2 |
    // resident head weights (wres)
    float* hs = reinterpret_cast<float*>(csm);
    uint64_t* pkey_s = reinterpret_cast<uint64_t*>(hs + NP * d);
    float* aslice = reinterpret_cast<float*>(pkey_s + NP * k);
    float* rslice = aslice + NP * F;
    float* sqf = rslice + NP * F;  // r^2 of this block's features, per child
    uint8_t* stg = reinterpret_cast<uint8_t*>(sqf + NP * F);
    const int stage_bytes = a.stage_bytes;
    uint64_t* kz = reinterpret_cast<uint64_t*>(stg + 2 * stage_bytes);
    float* xbuf = reinterpret_cast<float*>(kz + NP * a.R);
    // with a.wres: this block's W_i rows [F][2d] and W_o rows [F][d], kept
    // for the whole round (read at every depth)
    // the merged children lists of the nodes this block merged: [NP][k]
    float* nlq = xbuf + NP * d;
    int* ntok = reinterpret_cast<int*>(nlq + NP * k);
    float* dls = reinterpret_cast<float*>(ntok + NP * k);  // [R] the depth's drafter logits of the block's rows
    float* wis = reinterpret_cast<float*>((reinterpret_cast<uintptr_t>(dls + a.R) + 15) & ~static_cast<uintptr_t>(15));
    float* wos = wis + F * 2 * d;
    volatile int* abort = &misc[0];

    SelectArgs sa;
    sa.k = k;
    sa.W = a.W;
    sa.L = a.L;
    sa.nseq = a.nseq;
    sa.beta = a.beta;
    sa.node_logq = a.node_logq;
    sa.node_tok = a.node_tok;
    sa.node_lse = a.node_lse;
    sa.tree_tok = a.tree_tok;
    sa.tree_parent = a.tree_parent;
    sa.tree_score = a.tree_score;
    sa.tree_count = a.tree_count;
    sa.child_prow = a.child_prow;
    sa.child_tok = a.child_tok;
    sa.status = a.status;

    const int v0 = static_cast<int>((static_cast<long long>(rank) * a.V) / kCS);
    const int R = static_cast<int>((static_cast<long long>(rank + 1) * a.V) / kCS) - v0;
    const float4* hs4 = reinterpret_cast<const float4*>(hs);
    // the block's E rows stream through two stages of CR rows
    const int CR = stage_bytes / (d * 4);
    const int nch = (R + CR - 1) / CR;
    const uint8_t* esrc = reinterpret_cast<const uint8_t*>(a.E) + static_cast<size_t>(v0) * d * 4;
    // one stream of L * nch chunks (chunk g = chunk g % nch of depth g / nch
    // + 1) through stage g & 1, the stage's (g >> 1)-th use
    const int gtotal = a.L * nch;
    int issued = 0, consumed = 0;  // (thread 0's counts, for the drain after a timeout)
    auto issue = [&](int g) {  // thread 0
        issued = g + 1;
        const int ch = g % nch;
        const int rows = min(CR, R - ch * CR);
        const uint32_t bytes = static_cast<uint32_t>(rows) * d * 4;
        mbar_arrive_expect_tx(&sbar[g & 1], bytes);
        bulk_load(stg + (g & 1) * stage_bytes, esrc + static_cast<size_t>(ch) * CR * d * 4, bytes, &sbar[g & 1]);
    };
    if (tid == 0) {
        misc[0] = 0;
        mbar_init(&sbar[0], 1);
        mbar_init(&sbar[1], 1);
        mbar_init(&sbar[2], 1);
        fence_mbar_init();
    }
    __syncthreads();
    if (tid == 0) {
        for (int g = 0; g < 2 && g < gtotal; g++) issue(g);
        if (a.wres && a.L > 1) {
            const uint32_t bi = static_cast<uint32_t>(F) * 2 * d * 4, bo = static_cast<uint32_t>(F) * d * 4;
            mbar_arrive_expect_tx(&sbar[2], bi + bo);
            bulk_load(wis, a.Wi + static_cast<size_t>(rank) * F * 2 * d, bi, &sbar[2]);
            bulk_load(wos, a.Wo + static_cast<size_t>(rank) * F * d, bo, &sbar[2]);
        }
    }
    bool wready = false;

    for (int dep = 1; dep <= a.L; dep++) {
        const int P = a.caps[dep - 1], Pn = a.caps[dep];
        float* hcur = (dep & 1) ? a.h0 : a.h1;
        // the depth's drafter logits of this block's rows, requested first
        // (they arrive while the states are gathered)
        const float* drow = a.dlog + (static_cast<size_t>(s) * a.L + dep - 1) * a.V;
        constexpr int kDl = 8;  // R <= 8 * kRoundThreads
        float dlr[kDl];
#pragma unroll
        for (int u = 0; u < kDl; u++) {
            const int r = tid + u * kRoundThreads;
            dlr[u] = r < R ? __ldg(drow + v0 + r) : 0.0f;
        }
        // A1: the depth's states: the anchor, or r / rms(r) of the previous
        // depth's children gathered from the blocks that own the features
        if (dep == 1) {
            for (int j = tid; j < d; j += kRoundThreads) hs[j] = __ldg(a.anchor + static_cast<size_t>(s) * d + j);
        } else {
            for (int p = w; p < P; p += kRoundWarps) {
                float t = lane < kCS ? ld_cl_f32(&ssq_s[p], static_cast<uint32_t>(lane)) : 0.0f;
                t = warp_sum(t);
                const float sc = rsqrtf(t / static_cast<float>(d) + a.eps);
                constexpr int kB = 8;  // remote loads in flight per lane
                for (int j0 = 0; j0 < d; j0 += 32 * kB) {
                    float v[kB];
#pragma unroll
                    for (int u = 0; u < kB; u++) {
                        const int j = j0 + lane + 32 * u;
                        v[u] = j < d ? ld_cl_f32(&rslice[p * F + j % F], static_cast<uint32_t>(j / F)) : 0.0f;
                    }
#pragma unroll
                    for (int u = 0; u < kB; u++) {
                        const int j = j0 + lane + 32 * u;
                        if (j < d) hs[p * d + j] = v[u] * sc;
                    }
                }
            }
        }
#pragma unroll
        for (int u = 0; u < kDl; u++) {
            const int r = tid + u * kRoundThreads;
            if (r < R) dls[r] = dlr[u];
        }
        __syncthreads();
        for (int q = tid; q < P * F; q += kRoundThreads) {
            const int p = q / F, i = static_cast<int>(rank) * F + q % F;
            hcur[static_cast<size_t>(s * P + p) * d + i] = hs[p * d + i];
        }
        // A2: z of this block's rows for the P nodes: warps take RS rows at a
        // time, lanes split d; the partial sums are reduce-scattered.  Where
        // the nodes' states fit (NP * d/128 float4 per lane <= 8) each lane
        // keeps its share of them in registers for all chunks of the depth
        constexpr int kQR = NP <= 8 ? 8 / NP : 1;
        const bool hreg = NP <= 8 && d4 <= 32 * kQR;
        float4 hr[kQR * NP];
        if (hreg) {
#pragma unroll
            for (int qi = 0; qi < kQR; qi++) {
                const int q = lane + 32 * qi;
#pragma unroll
                for (int n = 0; n < NP; n++)
                    hr[qi * NP + n] = (q < d4 && n < P) ? hs4[n * d4 + q] : make_float4(0.f, 0.f, 0.f, 0.f);
            }
        }
        for (int ch = 0; ch < nch; ch++) {
            const int g = (dep - 1) * nch + ch;
            const int st = g & 1;
            const int rows = min(CR, R - ch * CR);
            if (!mbar_wait(&sbar[st], static_cast<uint32_t>(g >> 1) & 1u, abort)) {
                if (lane == 0) {
                    *abort = 1;
                    atomicOr(a.status, kDevTimeout);
                }
            } else {
                consumed = g + 1;
            }
            const float4* e4 = reinterpret_cast<const float4*>(stg + st * stage_bytes);
            for (int r0 = w * RS; r0 < rows; r0 += kRoundWarps * RS) {
                float v[32];
#pragma unroll
                for (int j = 0; j < 32; j++) v[j] = 0.0f;
                if (hreg) {
#pragma unroll
                    for (int qi = 0; qi < kQR; qi++) {
                        const int q = lane + 32 * qi;
                        if (q < d4) {
#pragma unroll
                            for (int r = 0; r < RS; r++) {
                                const float4 e = r0 + r < rows ? e4[(r0 + r) * d4 + q] : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                                for (int n = 0; n < NP; n++) v[r * NP + n] = dot4(e, hr[qi * NP + n], v[r * NP + n]);
                            }
                        }
                    }
                } else {
                    for (int q = lane; q < d4; q += 32) {
                        float4 hq[NP];
#pragma unroll
                        for (int n = 0; n < NP; n++) hq[n] = n < P ? hs4[n * d4 + q] : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                        for (int r = 0; r < RS; r++) {
                            const float4 e = r0 + r < rows ? e4[(r0 + r) * d4 + q] : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                            for (int n = 0; n < NP; n++) v[r * NP + n] = dot4(e, hq[n], v[r * NP + n]);
                        }
                    }
                }
                warp_reduce_scatter32(v, lane);
                const int r = lane / NP, n = lane % NP;
                const int row = ch * CR + r0 + r;
                if (n < P && r0 + r < rows) {
                    const int vv = v0 + row;
                    kz[n * a.R + row] = make_key((v[0] + dls[row]) * a.invT, static_cast<uint32_t>(vv));
                }
            }
            __syncthreads();  // stage st is free again
            if (tid == 0 && g + 2 < gtotal && !*abort) issue(g + 2);  // possibly the next depth's first chunks
        }
        // A3: per node, (max, sum exp) of the slice and its k best keys
        for (int p = w; p < P; p += kRoundWarps) {
            uint64_t* kn = kz + p * a.R;
            float m = -INFINITY;
            for (int i = lane; i < R; i += 32) m = fmaxf(m, key_val(kn[i]));
            m = warp_max(m);
            float sum = 0.0f;
            if (m != -INFINITY)
                for (int i = lane; i < R; i += 32) {
                    const float z = key_val(kn[i]);
                    if (z != -INFINITY) sum += __expf(z - m);
                }
            sum = warp_sum(sum);
            if (lane == 0) pms_s[p] = make_float2(m, sum);
            for (int j = 0; j < k; j++) {
                uint64_t best = 0ull;
                int at = -1;
                for (int i = lane; i < R; i += 32)
                    if (kn[i] > best) {
                        best = kn[i];
                        at = i;
                    }
                const uint64_t tp = warp_max_key(best);
                if (tp != 0ull && best == tp) kn[at] = 0ull;
                if (lane == 0) pkey_s[p * k + j] = tp;
                __syncwarp();
            }
        }
        cluster_sync_all();
        // B1: node p merged by block p % kCS, warp p / kCS
        const int prev_count = dep == 1 ? 1 : static_cast<int>(ld_cl_u32(&fcount, 0u));
        for (int p = static_cast<int>(rank) + kCS * w; p < P; p += kCS * kRoundWarps) {
            const int n = s * P + p;
            float* lq_out = a.node_logq + static_cast<size_t>(n) * k;
            int* tok_out = a.node_tok + static_cast<size_t>(n) * k;
            if (p >= prev_count) {
                for (int j = lane; j < k; j += 32) {
                    lq_out[j] = -INFINITY;
                    tok_out[j] = -1;
                }
                if (lane == 0) a.node_lse[n] = -INFINITY;
                continue;
            }
            float2 acc = lane < kCS ? ld_cl_f32x2(&pms_s[p], static_cast<uint32_t>(lane)) : make_float2(-INFINITY, 0.0f);
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                float2 other;
                other.x = __shfl_xor_sync(kFull, acc.x, o);
                other.y = __shfl_xor_sync(kFull, acc.y, o);
                acc = (lane & o) ? lse_merge(other, acc) : lse_merge(acc, other);
            }
            const float lse = acc.x == -INFINITY ? -INFINITY : acc.x + logf(acc.y);
            auto put = [&](int j, uint64_t tp) {
                const float z = tp != 0ull ? key_val(tp) : -INFINITY;
                const float lq = (lse != -INFINITY && z != -INFINITY) ? fminf(z - lse, 0.0f) : -INFINITY;
                const int tkn = tp != 0ull ? static_cast<int>(key_idx(tp)) : -1;
                lq_out[j] = lq;
                tok_out[j] = tkn;
                nlq[p * k + j] = lq;
                ntok[p * k + j] = tkn;
            };
            int ptr = 0;
            uint64_t head = lane < kCS ? ld_cl_u64(&pkey_s[p * k], static_cast<uint32_t>(lane)) : 0ull;
            uint64_t nxt = lane < kCS && k > 1 ? ld_cl_u64(&pkey_s[p * k + 1], static_cast<uint32_t>(lane)) : 0ull;
            for (int j = 0; j < k; j++) {
                const uint64_t tp = warp_max_key(head);
                if (tp != 0ull && head == tp) {
                    ptr++;
                    head = nxt;
                    nxt = ptr + 1 < k ? ld_cl_u64(&pkey_s[p * k + ptr + 1], static_cast<uint32_t>(lane)) : 0ull;
                }
                if (lane == 0) put(j, tp);
            }
            if (lane == 0) a.node_lse[n] = lse;
        }
        cluster_sync_all();
        // B2: the frontier (and after depth L prune and emit), rank 0
        if (rank == 0) {
            sa.N = a.nseq * P;
            sa.P = P;
            sa.dep = dep;
            sa.Pn = Pn;
            if (w == 0) select_frontier_cluster(sa, s, prev_count, nlq, ntok, fscore, cprow, ctokr, &fcount);
            if (dep == a.L) {
                __syncthreads();
                prune_emit_seq<kRoundThreads>(a.emit, s);
            }
        }
        if (dep == a.L) break;
        cluster_sync_all();
        // C1: a_c = SiLU(W_i [h_p ; E[t_c]]) for this block's features: the
        // children's E rows are staged first; 16 lanes per feature, each a
        // strided 1/16 of the row (coalesced), every child's partial sums
        // reduced over the 16 lanes
        if (tid < Pn) {
            const int pp = static_cast<int>(ld_cl_u32(&cprow[tid], 0u));
            const int tk = static_cast<int>(ld_cl_u32(&ctokr[tid], 0u));
            const bool ok = pp >= 0 && pp < P && static_cast<unsigned>(tk) < static_cast<unsigned>(a.V);
            (void)bounds_check(a.status, pp < 0 || ok);
            cpar[tid] = ok ? pp : -1;
            cpar_tok[tid] = ok ? tk : -1;
        }
        __syncthreads();
        for (int q = tid; q < Pn * d4; q += kRoundThreads) {
            const int c = q / d4, j = q % d4;
            const int tk = cpar_tok[c];
            reinterpret_cast<float4*>(xbuf)[q] =
                tk >= 0 ? __ldg(reinterpret_cast<const float4*>(a.E) + static_cast<size_t>(tk) * d4 + j)
                        : make_float4(0.f, 0.f, 0.f, 0.f);
        }
        if (a.wres && !wready) {
            if (!mbar_wait(&sbar[2], 0u, abort) && lane == 0) {
                *abort = 1;
                atomicOr(a.status, kDevTimeout);
            }
            wready = true;
        }
        __syncthreads();
        const float4* xb4 = reinterpret_cast<const float4*>(xbuf);
        const int sl = tid & 15;
        for (int il0 = 0; il0 < F; il0 += kRoundThreads / 16) {
            const int il = il0 + (tid >> 4);
            const bool fok = il < F;
            const float4* wr = reinterpret_cast<const float4*>(
                a.wres ? wis + static_cast<size_t>(fok ? il : 0) * 2 * d
                       : a.Wi + static_cast<size_t>(rank * F + (fok ? il : 0)) * 2 * d);
            float acc[NP];
            // each child's operand [h_p ; E[t_c]] as two row pointers, the
            // slot's parent read once (one shared-memory load per product)
            const float4* hrow[NP];
            const float4* xrow[NP];
            bool use[NP];
#pragma unroll
            for (int c = 0; c < NP; c++) {
                acc[c] = 0.0f;
                const int cp = c < Pn ? cpar[c] : -1;
                use[c] = cp >= 0;
                hrow[c] = hs4 + (cp >= 0 ? cp : 0) * d4;
                xrow[c] = xb4 + c * d4 - d4;
            }
            for (int q0 = sl; q0 < 2 * d4; q0 += 16 * 8) {
                float4 wv[8];
#pragma unroll
                for (int u = 0; u < 8; u++)
                    if (q0 + 16 * u < 2 * d4) wv[u] = wr[q0 + 16 * u];
#pragma unroll
                for (int u = 0; u < 8; u++) {
                    const int q = q0 + 16 * u;
                    if (q < 2 * d4) {
#pragma unroll
                        for (int c = 0; c < NP; c++) {
                            if (use[c]) acc[c] = dot4(wv[u], (q < d4 ? hrow[c] : xrow[c])[q], acc[c]);
                        }
                    }
                }
            }
#pragma unroll
            for (int c = 0; c < NP; c++) {
                float u = acc[c];
#pragma unroll
                for (int o = 8; o > 0; o >>= 1) u += __shfl_xor_sync(kFull, u, o);
                if (c < Pn && sl == 0 && fok) aslice[c * F + il] = cpar[c] >= 0 ? u / (1.0f + __expf(-u)) : 0.0f;
            }
        }
        cluster_sync_all();
        // C2: r_c = h_p + W_o a_c for this block's features, and their r^2
        for (int q = tid; q < Pn * d; q += kRoundThreads) {
            const int c = q / d, j = q % d;
            xbuf[q] = ld_cl_f32(&aslice[c * F + j % F], static_cast<uint32_t>(j / F));
        }
        __syncthreads();
        for (int il0 = 0; il0 < F; il0 += kRoundThreads / 16) {
            const int il = il0 + (tid >> 4);
            const bool fok = il < F;
            const int i = static_cast<int>(rank) * F + (fok ? il : 0);
            const float4* wr = reinterpret_cast<const float4*>(a.wres ? wos + static_cast<size_t>(fok ? il : 0) * d
                                                                       : a.Wo + static_cast<size_t>(i) * d);
            float acc[NP];
            bool use[NP];
#pragma unroll
            for (int c = 0; c < NP; c++) {
                acc[c] = 0.0f;
                use[c] = c < Pn && cpar[c] >= 0;
            }
            for (int q0 = sl; q0 < d4; q0 += 16 * 8) {
                float4 wv[8];
#pragma unroll
                for (int u = 0; u < 8; u++)
                    if (q0 + 16 * u < d4) wv[u] = wr[q0 + 16 * u];
#pragma unroll
                for (int u = 0; u < 8; u++) {
                    const int q = q0 + 16 * u;
                    if (q < d4) {
#pragma unroll
                        for (int c = 0; c < NP; c++)
                            if (use[c]) acc[c] = dot4(wv[u], xb4[c * d4 + q], acc[c]);
                    }
                }
            }
#pragma unroll
            for (int c = 0; c < NP; c++) {
                float y = acc[c];
#pragma unroll
                for (int o = 8; o > 0; o >>= 1) y += __shfl_xor_sync(kFull, y, o);
                if (c < Pn && sl == 0 && fok) {
                    const float r = cpar[c] >= 0 ? hs[cpar[c] * d + i] + y : 0.0f;
                    rslice[c * F + il] = r;
                    sqf[c * F + il] = r * r;
                }
            }
        }
        __syncthreads();
        for (int c = tid; c < Pn; c += kRoundThreads) {
            float t = 0.0f;
            for (int il = 0; il < F; il++) t += sqf[c * F + il];  // features in order
            ssq_s[c] = t;
        }
        cluster_sync_all();
    }
    if (tid == 0 && *abort) {
        // a wait gave up: the copies this block issued and did not consume
        // finish before it exits (their waits bounded again)
        int zero = 0;
        for (int g = consumed; g < issued; g++) (void)mbar_wait(&sbar[g & 1], static_cast<uint32_t>(g >> 1) & 1u, &zero);
        if (a.wres && a.L > 1) (void)mbar_wait(&sbar[2], 0u, &zero);
    }
    cluster_sync_all();  // no block leaves while a peer may still read its shared memory
}

// Two blocks wait at a grid barrier that expects three (test hook): each
// gives up after limit_ns, sets the timeout bit and the abort flag, and
// returns.  Nothing but the barrier words, the flag and the status word is
// touched.
__global__ void barrier_probe_kernel(unsigned* bar, int* abort, int* status, unsigned long long limit_ns) {
    __shared__ int sflag;
    (void)grid_barrier(bar, gridDim.x + 1, abort, status, &sflag, limit_ns);
}

template <int NM>
size_t round_smem_nm(int d, int R, int W, int k, int G, bool ecache, bool mstage) {
    const size_t es = ecache ? static_cast<size_t>(R) * (d + 4) * 4 : 0;
    const size_t a_part = static_cast<size_t>(NM) * d * 4 + static_cast<size_t>(kRoundWarps) * NM * 32 * 4 +
                          static_cast<size_t>(NM) * R * 8;
    const size_t b_part = static_cast<size_t>(W) * k * 12 + (kRankMax + 64) * 8 +
                          (mstage ? static_cast<size_t>(kRoundWarps) * G * k * 8 : 0);
    return es + (a_part > b_part ? a_part : b_part) + 16;
}

}  // namespace

template <int NP>
size_t round_cluster_smem_pm(int d, int R, int W, int k, int stage_bytes, bool wres) {
    (void)W;
    const int F = d / kCS;
    return static_cast<size_t>(NP) * d * 4 + static_cast<size_t>(NP) * k * 8 + 3 * static_cast<size_t>(NP) * F * 4 +
           2 * static_cast<size_t>(stage_bytes) + static_cast<size_t>(NP) * R * 8 + static_cast<size_t>(NP) * d * 4 +
           static_cast<size_t>(NP) * k * 8 + static_cast<size_t>(R) * 4 + 16 +
           (wres ? static_cast<size_t>(F) * 3 * d * 4 : 0);
}

int round_small_nm(int nmax) { return nmax <= 4 ? 4 : (nmax <= 8 ? 8 : (nmax <= 16 ? 16 : (nmax <= 32 ? 32 : 0))); }

size_t round_small_smem(int nm, int d, int R, int W, int k, int G, bool ecache, bool mstage) {
    switch (nm) {
        case 4: return round_smem_nm<4>(d, R, W, k, G, ecache, mstage);
        case 8: return round_smem_nm<8>(d, R, W, k, G, ecache, mstage);
        case 16: return round_smem_nm<16>(d, R, W, k, G, ecache, mstage);
        case 32: return round_smem_nm<32>(d, R, W, k, G, ecache, mstage);
        default: return 0;
    }
}

size_t round_cluster_smem(int pm, int d, int R, int W, int k, int stage_bytes, bool wres) {
    switch (pm) {
        case 4: return round_cluster_smem_pm<4>(d, R, W, k, stage_bytes, wres);
        case 8: return round_cluster_smem_pm<8>(d, R, W, k, stage_bytes, wres);
        case 16: return round_cluster_smem_pm<16>(d, R, W, k, stage_bytes, wres);
        case 32: return round_cluster_smem_pm<32>(d, R, W, k, stage_bytes, wres);
        default: return 0;
    }
}

static const void* round_cluster_kernel_of(int pm) {
    switch (pm) {
        case 4: return reinterpret_cast<const void*>(round_cluster_f32_kernel<4>);
        case 8: return reinterpret_cast<const void*>(round_cluster_f32_kernel<8>);
        case 16: return reinterpret_cast<const void*>(round_cluster_f32_kernel<16>);
        case 32: return reinterpret_cast<const void*>(round_cluster_f32_kernel<32>);
        default: return nullptr;
    }
}

cudaError_t round_cluster_set_attributes() {
    cudaError_t e = cudaSuccess;
    for (int pm : {4, 8, 16, 32}) {
        const void* fn = round_cluster_kernel_of(pm);
        if (e == cudaSuccess) e = set_max_dynamic_smem(fn);
        if (e == cudaSuccess) e = cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    }
    return e;
}

size_t round_cluster_static_smem(int pm) {
    cudaFuncAttributes fa;
    const void* fn = round_cluster_kernel_of(pm);
    if (!fn || cudaFuncGetAttributes(&fa, fn) != cudaSuccess) return 64 * 1024;
    return fa.sharedSizeBytes;
}

// Whether a cluster of kCS blocks with `smem` bytes each can be scheduled.
bool round_cluster_fits(int pm, size_t smem) {
    const void* fn = round_cluster_kernel_of(pm);
    if (!fn) return false;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(kCS);
    cfg.blockDim = dim3(kRoundThreads);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = kCS;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    return cudaOccupancyMaxActiveClusters(&n, fn, &cfg) == cudaSuccess && n >= 1;
}

cudaError_t launch_round_cluster_f32(const RoundArgs& a, int pm, size_t smem, cudaStream_t st) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(a.nseq * kCS);
    cfg.blockDim = dim3(kRoundThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = kCS;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    switch (pm) {
        case 4: return cudaLaunchKernelEx(&cfg, round_cluster_f32_kernel<4>, a);
        case 8: return cudaLaunchKernelEx(&cfg, round_cluster_f32_kernel<8>, a);
        case 16: return cudaLaunchKernelEx(&cfg, round_cluster_f32_kernel<16>, a);
        case 32: return cudaLaunchKernelEx(&cfg, round_cluster_f32_kernel<32>, a);
        default: return cudaErrorInvalidValue;
    }
}

static const void* round_kernel_of(int nm) {
    switch (nm) {
        case 4: return reinterpret_cast<const void*>(round_small_f32_kernel<4>);
        case 8: return reinterpret_cast<const void*>(round_small_f32_kernel<8>);
        case 16: return reinterpret_cast<const void*>(round_small_f32_kernel<16>);
        case 32: return reinterpret_cast<const void*>(round_small_f32_kernel<32>);
        default: return nullptr;
    }
}

cudaError_t round_small_set_smem_limits() {
    cudaError_t e = cudaSuccess;
    for (int nm : {4, 8, 16, 32})
        if (e == cudaSuccess) e = set_max_dynamic_smem(round_kernel_of(nm));
    return e;
}

int round_small_blocks_per_sm(int nm, size_t smem) {
    int n = 0;
    const void* fn = round_kernel_of(nm);
    if (!fn || cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, fn, kRoundThreads, smem) != cudaSuccess) return 0;
    return n;
}

cudaError_t launch_barrier_probe(unsigned* bar, int* abort, int* status, unsigned long long limit_ns,
                                 cudaStream_t st) {
    barrier_probe_kernel<<<2, 32, 0, st>>>(bar, abort, status, limit_ns);
    return cudaGetLastError();
}

cudaError_t launch_round_small_f32(const RoundArgs& a, int nm, size_t smem, cudaStream_t st) {
    const void* fn = round_kernel_of(nm);
    if (!fn) return cudaErrorInvalidValue;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(a.G);
    cfg.blockDim = dim3(kRoundThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    switch (nm) {
        case 4: return cudaLaunchKernelEx(&cfg, round_small_f32_kernel<4>, a);
        case 8: return cudaLaunchKernelEx(&cfg, round_small_f32_kernel<8>, a);
        case 16: return cudaLaunchKernelEx(&cfg, round_small_f32_kernel<16>, a);
        default: return cudaLaunchKernelEx(&cfg, round_small_f32_kernel<32>, a);
    }
}

}  // namespace dart
