// fe_lm_head_topk_noalloc: the LM head with its fused softmax statistics and top-k, for
// callers that cannot allocate device memory.
//
// Some callers cannot call cudaMalloc at the point where they need this step: code that
// runs while a memory pool or arena is frozen, code inside a host callback or a custom
// allocator's own path, or a runtime that budgets every allocation up front and forbids
// new ones on the serving path. This entry point allocates nothing. It reads the LM head
// (and final RMSNorm gain) that fe_draft_init already packed into the handle, takes the
// hidden rows and the outputs from the caller, and keeps its working memory (per-slab
// partial results, completion counters and the tensor-core operand) in one file-scope
// __device__ array of a fixed size, held until the process exits.
//
// When the array is reserved: fe_draft_init looks up its device address with
// cudaGetSymbolAddress, once per device, with that device current. Under CUDA's lazy
// module loading (the default since CUDA 12.2, CUDA_MODULE_LOADING=LAZY) that lookup is
// what loads this file's module and reserves the array, so the memory is taken inside
// fe_draft_init, which allocates anyway; with CUDA_MODULE_LOADING=EAGER it is reserved
// when the library's modules load on the device. Either way no call of
// fe_lm_head_topk_noalloc allocates or looks anything up.
//
// Limits: at most kMaxRows hidden rows (n_layers * B), d <= kMaxD, top_k <= 32.
// Sharing: every call uses the same array and leaves its contents behind. Calls that may
// overlap on the GPU (different streams, or different host threads) race with each other
// and must be serialised by the caller. The completion counters, which must start at
// zero, are cleared by every call.
// Device: the call must be made with the handle's device current (the array, the LM head
// and the status word it uses all live there); otherwise it returns FE_ERR_INVALID_ARG.
#include <cstdio>
#include <mutex>

#include "fe_kernels.h"

namespace {

constexpr int kMaxRows = 16;     // hidden rows (n_layers * B) per call
constexpr int kMaxSlabs = 256;   // vocabulary slabs (CTAs) of the LM-head kernels
constexpr int kMaxTopK = 32;
constexpr int kMaxD = 16384;
constexpr int kMaxDevices = 64;

constexpr size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }
constexpr size_t kPartIdBytes = align256((size_t)kMaxRows * kMaxSlabs * kMaxTopK * 4);
constexpr size_t kPartValBytes = align256((size_t)kMaxRows * kMaxSlabs * kMaxTopK * 4);
constexpr size_t kPartMsBytes = align256((size_t)kMaxRows * kMaxSlabs * 2 * 4);
constexpr size_t kCounterBytes = align256((size_t)kMaxRows * 4);
constexpr size_t kOperandBytes = align256((size_t)2 * kMaxRows * kMaxD * 2);  // bf16 hi/lo rows
constexpr size_t kScratchBytes = kPartIdBytes + kPartValBytes + kPartMsBytes + kCounterBytes + kOperandBytes;

// ~2.1 MB on every device that loads the library, for the life of the process.
static __device__ __align__(256) unsigned char g_scratch[kScratchBytes];

std::mutex g_mu;
unsigned char* g_scratch_dev[kMaxDevices] = {};  // device address of g_scratch, per device

}  // namespace

using namespace fe;

cudaError_t fe::noalloc_resolve_scratch(int device) {
    if (device < 0 || device >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_mu);
    if (g_scratch_dev[device]) return cudaSuccess;
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_scratch);
    if (e != cudaSuccess) return e;
    if (!p) return cudaErrorInvalidSymbol;
    g_scratch_dev[device] = (unsigned char*)p;
    return cudaSuccess;
}

extern "C" FE_API fe_status fe_lm_head_topk_noalloc(fe_handle* h, const float* hidden, int32_t B, int32_t top_k,
                                                    float temperature, int32_t* topk_id, float* topk_logit,
                                                    float* topk_prob, float* lse, void* stream) {
    LmHeadView v;
    if (!handle_lmhead_view(h, &v) || !hidden || !topk_id || !topk_logit || !topk_prob || !lse)
        return FE_ERR_INVALID_ARG;
    if (reinterpret_cast<uintptr_t>(hidden) & 15) return FE_ERR_INVALID_ARG;  // read as 16-byte vectors
    if (B < 1 || B > v.max_batch || top_k < 1 || top_k > v.top_k_max || top_k > kMaxTopK)
        return FE_ERR_INVALID_ARG;
    if (!(temperature == temperature)) return FE_ERR_INVALID_ARG;
    const int R = v.N * B;
    char msg[200];
    if (R > kMaxRows || v.d > kMaxD) {
        snprintf(msg, sizeof(msg),
                 "fe_lm_head_topk_noalloc: n_layers*B = %d (max %d) or d = %d (max %d) exceeds its fixed scratch", R,
                 kMaxRows, v.d, kMaxD);
        set_error_detail(msg);
        return FE_ERR_INVALID_ARG;
    }
    if (v.n_slabs > kMaxSlabs) {
        snprintf(msg, sizeof(msg),
                 "fe_lm_head_topk_noalloc: the LM head's %d vocabulary slabs exceed its fixed scratch (max %d)",
                 v.n_slabs, kMaxSlabs);
        set_error_detail(msg);
        return FE_ERR_INVALID_ARG;
    }
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess) return FE_ERR_CUDA;
    if (dev != v.device) {
        snprintf(msg, sizeof(msg), "fe_lm_head_topk_noalloc: the current CUDA device (%d) is not the handle's (%d)",
                 dev, v.device);
        set_error_detail(msg);
        return FE_ERR_INVALID_ARG;
    }
    unsigned char* base = nullptr;
    {
        std::lock_guard<std::mutex> lock(g_mu);
        base = dev >= 0 && dev < kMaxDevices ? g_scratch_dev[dev] : nullptr;
    }
    if (!base) {  // fe_draft_init resolved it for the handle's device; this does not happen
        set_error_detail("fe_lm_head_topk_noalloc: the scratch array was not resolved for this device");
        return FE_ERR_CUDA;
    }
    cudaStream_t st = (cudaStream_t)stream;
    LmHeadArgs lm{};
    lm.W = v.lm_head;
    lm.gamma = v.final_norm;
    lm.V = v.V;
    lm.d = v.d;
    lm.R = R;
    lm.B = B;
    lm.N = v.N;
    lm.hid = hidden;
    lm.eps = v.eps;
    lm.inv_temp = temperature > 0.f ? 1.0f / temperature : 1.0f;
    lm.top_k = top_k;
    lm.n_slabs = v.n_slabs;
    lm.part_id = (int*)base;
    lm.part_val = (float*)(base + kPartIdBytes);
    lm.part_ms = (float*)(base + kPartIdBytes + kPartValBytes);
    lm.counters = (int*)(base + kPartIdBytes + kPartValBytes + kPartMsBytes);
    lm.dbg_logits = nullptr;
    lm.topk_id = topk_id;
    lm.topk_logit = topk_logit;
    lm.topk_prob = topk_prob;
    lm.lse = lse;
    lm.status = v.status;
    lm.pdl = false;
    uint16_t* operand = (uint16_t*)(base + kPartIdBytes + kPartValBytes + kPartMsBytes + kCounterBytes);
    // the counters must start at zero (a call that ended early could have left them set)
    if (cudaMemsetAsync(lm.counters, 0, kCounterBytes, st) != cudaSuccess) return FE_ERR_CUDA;
    const cudaError_t e = v.mma ? launch_lmhead_mma(lm, operand, v.dev, st) : launch_lmhead(v.dtype, lm, v.dev, st);
    return e == cudaSuccess ? FE_OK : FE_ERR_CUDA;
}
