// dart_expand_root_noalloc: the depth-1 expansion (scoring of every root's
// children over the full vocabulary with the tensor-core LM-head kernel, the
// merge of its per-CTA partials and the selection of S_1) without any device
// allocation.  It exists for callers that must not allocate device memory
// while they run this step: an inference server that has handed all free
// memory to its own pool (KV cache, activations) and forbids further
// cudaMalloc, code running where cudaMalloc's implicit device
// synchronisation is unacceptable, or a host application whose allocator owns
// every device byte.  Such callers pass inputs and outputs; everything else
// lives in one file-scope device array, g_scratch, that every GPU loading
// this library holds until the process exits.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <mutex>

#include "../../include/dart.h"
#include "dart_device.cuh"
#include "dart_kernels.h"

using namespace dart;

namespace {

constexpr size_t kScratchBytes = size_t(16) << 20;  // 16 MiB per device
constexpr int kMaxSeqNoAlloc = 64;                  // roots per call
constexpr int kMaxDNoAlloc = 8192;                  // hidden size
constexpr int kBhalfNoAlloc = 64;                   // row offset of the lo half of the root states
constexpr int kMaxDevices = 64;

// Scratch shared by every call on a device.  Host code must not use this name
// as an address: the per-device address comes from cudaGetSymbolAddress.
__device__ __align__(256) unsigned char g_scratch[kScratchBytes];

struct DeviceSetup {
    bool ready;
    bool called;          // a call was enqueued on this device (its status word is meaningful)
    unsigned char* base;  // device address of g_scratch on this device
    int sms, optin;
};
DeviceSetup g_setup[kMaxDevices];
std::mutex g_setup_mu;

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn lookup_encode_tiled() {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
        return reinterpret_cast<EncodeTiledFn>(p);
    return nullptr;
}

// Looked up once; the initialisation of a function-local static is
// thread-safe, so first calls from several threads (on any devices) agree.
EncodeTiledFn encode_tiled() {
    static const EncodeTiledFn fn = lookup_encode_tiled();
    return fn;
}

bool encode_rows(CUtensorMap* m, const void* base, uint64_t inner, uint64_t rows, uint32_t box_rows) {
    EncodeTiledFn fn = encode_tiled();
    if (!fn) return false;
    cuuint64_t dims[2] = {inner, rows};
    cuuint64_t strides[1] = {inner * 2};
    cuuint32_t box[2] = {static_cast<cuuint32_t>(kBlockK), box_rows};
    cuuint32_t estr[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Once per device, with that device current: the scratch address and the
// kernels' shared-memory limits.
int setup_device(int dev, DeviceSetup* out) {
    if (dev < 0 || dev >= kMaxDevices) return DART_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_setup_mu);
    DeviceSetup& s = g_setup[dev];
    if (!s.ready) {
        int major = 0, minor = 0, sms = 0, optin = 0;
        if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess)
            return DART_ERR_CUDA;
        if (major != 10 || minor != 3) return DART_ERR_UNSUPPORTED;
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_scratch) != cudaSuccess || p == nullptr) return DART_ERR_CUDA;
        if (tc_set_smem_limits(optin) != cudaSuccess || select_set_smem_limits() != cudaSuccess)
            return DART_ERR_CUDA;
        s.base = static_cast<unsigned char*>(p);
        s.sms = sms;
        s.optin = optin;
        s.ready = true;
    }
    *out = s;
    return DART_OK;
}

size_t round256(size_t x) { return (x + 255) & ~size_t(255); }

}  // namespace

extern "C" int dart_expand_root_noalloc(const dart_config* cfg, const void* E, const float* drafter_logits,
                                        const float* anchor_h, int32_t* node_tok, float* node_logq, float* node_lse,
                                        int32_t* front_tok, float* front_score, int32_t* front_count,
                                        void* stream) {
    if (!cfg || !E || !drafter_logits || !anchor_h || !node_tok || !node_logq || !node_lse || !front_tok ||
        !front_score || !front_count)
        return DART_ERR_INVALID;
    const dart_config c = *cfg;
    // the problem limits of dart_init_head (nseq*W excepted: only depth 1 runs), plus this entry point's own
    if (c.V < 1 || c.V >= (1 << 24) || c.d < 64 || c.d % 64 || c.L < 1 || c.W < 1 || c.W > 64 ||
        c.L * c.W > 1024 || c.k < 1 || c.k > 64 || c.k > c.V || c.W * c.k > 4096 || c.B < 1 || c.B > 1024 ||
        c.nseq < 1 || !(c.beta <= 0.0f) || !std::isfinite(c.beta) || !(c.temperature >= 0.0f) ||
        !std::isfinite(c.temperature))
        return DART_ERR_INVALID;
    if (c.nseq > kMaxSeqNoAlloc || c.d > kMaxDNoAlloc) return DART_ERR_INVALID;
    if (c.cand_k != 0) return DART_ERR_INVALID;  // full-vocabulary scoring only
    if (c.lmhead_ctas_per_sm < 0 || c.lmhead_ctas_per_sm > 2) return DART_ERR_INVALID;
    if ((reinterpret_cast<uintptr_t>(E) & 15u) || (reinterpret_cast<uintptr_t>(drafter_logits) & 3u) ||
        (reinterpret_cast<uintptr_t>(anchor_h) & 15u))
        return DART_ERR_INVALID;

    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return DART_ERR_CUDA;
    DeviceSetup ds;
    int rc = setup_device(dev, &ds);
    if (rc != DART_OK) return rc;
    // kernel attributes are process-wide: re-apply the device maxima (no call lowers them)
    if (tc_set_smem_limits(ds.optin) != cudaSuccess || select_set_smem_limits() != cudaSuccess)
        return DART_ERR_CUDA;

    // launch plan of depth 1: the handle path's plan (plan_lmhead_tc) for N roots
    // and a row-major E (this entry point keeps no tiled copy)
    const int N = c.nseq;
    LmheadPlan lp;
    if (!plan_lmhead_tc(N, c.V, c.d, c.k, ds.sms, ds.optin, c.lmhead_ctas_per_sm, false, &lp) || lp.G != 1)
        return DART_ERR_UNSUPPORTED;
    const int NG = lp.NG, nV = lp.nV;
    const int tiles = (c.V + kTileM - 1) / kTileM;
    const int Pn = std::min(c.W, c.k);

    // carve the scratch array (the status word first, at a fixed offset that
    // dart_noalloc_status reads); reject sizes beyond it
    size_t off = 0;
    int* status = reinterpret_cast<int*>(ds.base);
    off += 256;
    auto take = [&](size_t bytes) {
        unsigned char* p = ds.base + off;
        off += round256(bytes);
        return p;
    };
    float* h32 = reinterpret_cast<float*>(take(size_t(N) * c.d * 4));
    __nv_bfloat16* HL = reinterpret_cast<__nv_bfloat16*>(take(size_t(2) * kBhalfNoAlloc * c.d * 2));
    float2* part_ms = reinterpret_cast<float2*>(take(size_t(nV) * N * 8));
    uint64_t* part_key = reinterpret_cast<uint64_t*>(take(size_t(N) * part_stride(nV, c.k) * 8));
    int* tree_parent = reinterpret_cast<int*>(take(size_t(N) * c.W * 4));
    int* child_prow = reinterpret_cast<int*>(take(size_t(N) * Pn * 4));
    int* child_tok = reinterpret_cast<int*>(take(size_t(N) * Pn * 4));
    int* seq_ticket = reinterpret_cast<int*>(take(size_t(N) * 4));
    uint64_t* gthr = reinterpret_cast<uint64_t*>(take(size_t(N) * 8));
    if (off > kScratchBytes) return DART_ERR_INVALID;

    CUtensorMap tmE, tmH;
    if (!encode_rows(&tmE, E, c.d, c.V, kTileM) || !encode_rows(&tmH, HL, c.d, 2 * kBhalfNoAlloc, NG))
        return DART_ERR_UNSUPPORTED;

    cudaStream_t st = static_cast<cudaStream_t>(stream);
    // the shared array keeps the previous call's contents: zero what must start at zero
    if (cudaMemsetAsync(seq_ticket, 0, size_t(N) * 4, st) != cudaSuccess ||
        cudaMemsetAsync(status, 0, 4, st) != cudaSuccess)
        return DART_ERR_CUDA;
    if (launch_prep_anchor(anchor_h, N, c.d, h32, HL, kBhalfNoAlloc, gthr, N, st) != cudaSuccess) return DART_ERR_CUDA;

    LmheadArgs la;
    std::memset(&la, 0, sizeof la);
    la.V = c.V;
    la.d = c.d;
    la.N = N;
    la.NG = NG;
    la.G = 1;
    la.nV = nV;
    la.k = c.k;
    la.tiles = tiles;
    la.P = 1;
    la.invT = c.temperature > 0.0f ? 1.0f / c.temperature : 1.0f;
    la.dlog = drafter_logits;
    la.dlog_seq_stride = static_cast<long long>(c.L) * c.V;
    la.dlog_row_off = 0;
    la.bhalf = kBhalfNoAlloc;
    la.stages = lp.stages;
    la.part_ms = part_ms;
    la.part_key = part_key;
    la.status = status;
    la.gthr = gthr;
    if (launch_lmhead_tc(&tmE, &tmH, la, lp.smem, st) != cudaSuccess) return DART_ERR_CUDA;

    SelectArgs sa;
    std::memset(&sa, 0, sizeof sa);
    sa.N = N;
    sa.P = 1;
    sa.k = c.k;
    sa.nV = nV;
    sa.klist = c.k;
    sa.W = c.W;
    sa.L = 1;
    sa.nseq = N;
    sa.dep = 1;
    sa.Pn = Pn;
    sa.beta = c.beta;
    sa.part_ms = part_ms;
    sa.part_key = part_key;
    sa.gthr = gthr;
    sa.node_logq = node_logq;
    sa.node_tok = node_tok;
    sa.node_lse = node_lse;
    sa.tree_tok = front_tok;
    sa.tree_parent = tree_parent;
    sa.tree_score = front_score;
    sa.tree_count = front_count;
    sa.child_prow = child_prow;
    sa.child_tok = child_tok;
    sa.seq_ticket = seq_ticket;
    sa.status = status;
    if (launch_merge_select(sa, st) != cudaSuccess) return DART_ERR_CUDA;
    {
        std::lock_guard<std::mutex> lock(g_setup_mu);
        g_setup[dev].called = true;
    }
    return DART_OK;
}

extern "C" int dart_noalloc_status(void* stream) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return DART_ERR_CUDA;
    if (dev < 0 || dev >= kMaxDevices) return DART_ERR_UNSUPPORTED;
    unsigned char* base = nullptr;
    {
        std::lock_guard<std::mutex> lock(g_setup_mu);
        if (!g_setup[dev].ready || !g_setup[dev].called) return DART_ERR_STATE;
        base = g_setup[dev].base;
    }
    if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return DART_ERR_CUDA;
    int word = 0;  // a pageable host int: cudaMemcpy stages it without allocating device memory
    if (cudaMemcpy(&word, base, sizeof word, cudaMemcpyDeviceToHost) != cudaSuccess) return DART_ERR_CUDA;
    return (word & kDevTimeout) ? DART_ERR_TIMEOUT : DART_OK;
}
