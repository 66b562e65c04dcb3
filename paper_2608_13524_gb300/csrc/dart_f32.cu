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

// LM-head scoring, fp32: one block of 128 threads (the 4 epilogue warps) per
// vocabulary range and node group; thread r owns row r of each 128-row tile.
template <int NG>
__global__ void __launch_bounds__(kEpiThreads) lmhead_f32_kernel(const LmheadArgs a) {
    extern __shared__ float smf[];
    pdl_trigger();
    pdl_wait();
    float* Es = smf;                     // [128][65]
    float* Hs = Es + kTileM * kEPad;     // [NG][64]
    EpiSmem e;
    e.cap = kCandCap;  // a whole tile: every candidate always fits
    e.list = reinterpret_cast<uint64_t*>(Hs + NG * kBlockK);
    e.cand = e.list + NG * a.k;
    e.gcache = e.cand + NG * kCandCap;
    e.stats = reinterpret_cast<float2*>(e.gcache + NG);
    e.mref = reinterpret_cast<float*>(e.stats + 4 * NG);
    e.cnt = reinterpret_cast<int*>(e.mref + 4 * NG);
    e.more = e.cnt + NG;

    const int g = blockIdx.x % a.G;
    const int vr = blockIdx.x / a.G;
    const int t0 = static_cast<int>((static_cast<long long>(vr) * a.tiles) / a.nV);
    const int t1 = static_cast<int>((static_cast<long long>(vr + 1) * a.tiles) / a.nV);
    const int tid = threadIdx.x, lane = tid & 31, ew = tid >> 5;
    const int KB = a.d / kBlockK;
    epi_init(e, NG, a.k, tid, kEpiThreads);
    float ssum[NG / 16];
#pragma unroll
    for (int c = 0; c < NG / 16; c++) ssum[c] = 0.0f;

    for (int t = t0; t < t1; t++) {
        float acc[NG];
#pragma unroll
        for (int j = 0; j < NG; j++) acc[j] = 0.0f;
        for (int kb = 0; kb < KB; kb++) {
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
            for (int q = tid; q < NG * kBlockK; q += kEpiThreads) {
                const int nn = q / kBlockK, c = q % kBlockK;
                const int n = g * NG + nn;
                Hs[q] = n < a.N ? a.h32[static_cast<size_t>(n) * a.d + kb * kBlockK + c] : 0.0f;
            }
            named_bar_sync(kEpiBarrier, kEpiThreads);
            const float* er = Es + tid * kEPad;
            for (int kk = 0; kk < kBlockK; kk++) {
                const float ev = er[kk];
#pragma unroll
                for (int j = 0; j < NG; j++) acc[j] = fmaf(ev, Hs[j * kBlockK + kk], acc[j]);
            }
        }
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
                if (n < a.N) {
                    nodemask |= 1u << j;
                    const int seq = n / a.P;
                    if (seq != cur_seq) {
                        cur_seq = seq;
                        const long long off = a.dlog_row ? static_cast<long long>(__ldg(a.dlog_row + seq)) * a.V
                                                         : a.dlog_row_off;
                        dl = valid ? __ldg(a.dlog + seq * a.dlog_seq_stride + off + v) : 0.0f;
                    }
                    z[j] = (acc[c0 + j] + dl) * a.invT;
                    if (a.zout && valid) a.zout[static_cast<long long>(n) * a.zout_stride + v] = z[j];
                }
            }
            (void)epi_chunk(e, NG, a.k, ew, lane, c0, z, nodemask, valid, static_cast<uint32_t>(v), ssum[c0 / 16]);
        }
        epi_merge(e, NG, a.k, ew, lane, kEpiThreads, tid, a.gthr, g * NG, a.N);
    }
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

template <int NG>
int smem_ng(int k) {
    return (kTileM * kEPad + NG * kBlockK) * 4 + NG * k * 8 + NG * kCandCap * 8 + NG * 8 + 4 * NG * 8 + 4 * NG * 4 + NG * 4 +
           8;
}

}  // namespace

int lmhead_f32_smem(int NG, int k) { return NG <= 16 ? smem_ng<16>(k) : smem_ng<32>(k); }

cudaError_t f32_set_smem_limits(int max_dyn) {
    cudaError_t e = cudaFuncSetAttribute(lmhead_f32_kernel<16>, cudaFuncAttributeMaxDynamicSharedMemorySize, max_dyn);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(lmhead_f32_kernel<32>, cudaFuncAttributeMaxDynamicSharedMemorySize, max_dyn);
    return e;
}

cudaError_t launch_lmhead_f32(const LmheadArgs& a, cudaStream_t st) {
    const int smem = lmhead_f32_smem(a.NG, a.k);
    if (a.NG == 16) return launch_pdl(lmhead_f32_kernel<16>, dim3(a.nV * a.G), dim3(kEpiThreads), smem, st, a);
    if (a.NG == 32) return launch_pdl(lmhead_f32_kernel<32>, dim3(a.nV * a.G), dim3(kEpiThreads), smem, st, a);
    return cudaErrorInvalidValue;
}

cudaError_t launch_gemm_f32(const GemmArgs& a, cudaStream_t st) {
    return launch_pdl(gemm_f32_kernel, dim3(a.MT * a.G * a.S), dim3(256), 0, st, a);
}

}  // namespace dart
