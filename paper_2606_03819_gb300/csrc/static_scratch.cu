// tf_stage1_marginals_static: the stage-1 LM-head top-k of tf_stage1_marginals for callers that
// cannot allocate device memory, with its scratch in a fixed array that the library itself
// holds on every GPU it is loaded on.
//
// Who needs it: code that runs inside a host framework that owns all device memory and gives its
// plugins or custom operators no workspace and no allocator, and code on a latency-critical path
// where cudaMalloc / cudaFree are ruled out because they can synchronise the whole device. Such
// a caller can pass inputs and outputs but cannot provide the workspace of tf_workspace_size.
//
// What it costs: kScratchBytes of device memory on every GPU that loads the library, held until
// the process exits, whether or not this entry point is ever called.
//
// The kernels are the ones tf_stage1_marginals runs (same launchers, same arguments); only the
// place of the per-block partials and of the status word differs.
#include <cuda.h>

#include <mutex>

#include "common.cuh"

namespace {

using namespace tf;

constexpr size_t kScratchBytes = TF_STATIC_SCRATCH_BYTES;
constexpr size_t kStatusBytes = 256;  // status word, padded so that the partials stay 256-byte aligned
constexpr int kMaxDevices = 64;

static_assert(kScratchBytes % 256 == 0 && kScratchBytes > kStatusBytes, "scratch size");

// The scratch: the status word at offset 0, then the LM-head partials (half-block summaries, then
// chunk records, each [n_tiles][part][rows]). Every call
// on a device shares it and it keeps whatever the last call left, so each call clears the status
// word before its first kernel; the partials need no clearing (the LM-head pass writes every
// entry the merge reads). In host code `g_scratch` names a host-side shadow of the symbol, not
// the device memory: host code must use the address cudaGetSymbolAddress returns instead.
static __device__ __align__(256) uint8_t g_scratch[kScratchBytes];

// The context a device address belongs to: the driver's unique id of the calling thread's
// current context (cuCtxGetCurrent + cuCtxGetId, reached through the runtime's driver entry
// points). A device reset or a re-created primary context gives a new id, and with it a new
// lookup of the array's address. Returns false if the driver offers no such id.
typedef CUresult (*CtxGetCurrentFn)(CUcontext*);
typedef CUresult (*CtxGetIdFn)(CUcontext, unsigned long long*);
bool current_context_id(unsigned long long* id) {
    static const CtxGetCurrentFn get_current = [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess)
            p = nullptr;
        return reinterpret_cast<CtxGetCurrentFn>(p);
    }();
    static const CtxGetIdFn get_id = [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess)
            p = nullptr;
        return reinterpret_cast<CtxGetIdFn>(p);
    }();
    CUcontext ctx = nullptr;
    if (!get_current || !get_id || get_current(&ctx) != CUDA_SUCCESS || !ctx) return false;
    return get_id(ctx, id) == CUDA_SUCCESS;
}

std::mutex g_setup_mutex;
void* g_scratch_addr[kMaxDevices] = {};
unsigned long long g_scratch_ctx[kMaxDevices] = {};

// Device address of g_scratch on the current device `dev`: looked up once per device and
// context (under a lock, so threads may race to the first call) and kept. Without a context id
// from the driver it is looked up on every call, which allocates nothing either.
tf_status scratch_address(int dev, uint8_t** out) {
    if (dev < 0 || dev >= kMaxDevices) return TF_ERR_UNSUPPORTED;
    // No current context yet (this thread's first runtime call on the device): the lookup below
    // binds the runtime's primary context, and the id is read after it.
    unsigned long long ctx = 0;
    bool have_ctx = current_context_id(&ctx);
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    if (!have_ctx || !g_scratch_addr[dev] || g_scratch_ctx[dev] != ctx) {
        void* p = nullptr;
        const cudaError_t e = cudaGetSymbolAddress(&p, g_scratch);
        if (e != cudaSuccess || !p) {
            (void)cudaGetLastError();  // do not leave the error for a later launch check to find
            return TF_ERR_CUDA;
        }
        if (!have_ctx) have_ctx = current_context_id(&ctx);
        g_scratch_addr[dev] = have_ctx ? p : nullptr;   // no id: look it up again next call
        g_scratch_ctx[dev] = ctx;
        *out = static_cast<uint8_t*>(p);
        return TF_OK;
    }
    *out = static_cast<uint8_t*>(g_scratch_addr[dev]);
    return TF_OK;
}

bool aligned16(const void* p) { return p && reinterpret_cast<uintptr_t>(p) % 16 == 0; }

tf_status from_cuda(cudaError_t e) { return e == cudaSuccess ? TF_OK : TF_ERR_CUDA; }

}  // namespace

extern "C" tf_status tf_stage1_marginals_static(const tf_dims* dims, const tf_weights* w, const void* hidden,
                                                int32_t* top_ids, float* top_logp, int32_t* dev_status,
                                                tf_stream_t stream) {
    // the same validation as every workspace call (host only)
    size_t ws_bytes = 0;
    const tf_status vs = tf_workspace_size(dims, &ws_bytes);
    if (vs != TF_OK) return vs;
    const int rows = dims->batch * dims->gamma;
    const int n_tiles = (dims->V + kBlockV - 1) / kBlockV;
    const int K1 = dims->M > dims->K2 ? dims->M : dims->K2;
    const float inv_temp = 1.0f / dims->temperature;
    // the scratch limit, then the pointers; both before any GPU work
    const size_t row_blocks = static_cast<size_t>(rows) * n_tiles;
    const size_t halves_bytes = (row_blocks * kHalfBytesPerRowBlock + 255) / 256 * 256;
    if (kStatusBytes + halves_bytes + row_blocks * kChunkBytesPerRowBlock > kScratchBytes)
        return TF_ERR_UNSUPPORTED;
    if (!w || !aligned16(w->lm_head) || !aligned16(hidden) || !top_ids || !top_logp || !dev_status)
        return TF_ERR_INVALID_ARG;

    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return TF_ERR_CUDA;
    uint8_t* scratch = nullptr;
    const tf_status ss = scratch_address(dev, &scratch);
    if (ss != TF_OK) return ss;
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 1)
        return TF_ERR_CUDA;

    const Ctx ctx{reinterpret_cast<cudaStream_t>(stream), sms, reinterpret_cast<int*>(scratch)};
    const Partials partials{reinterpret_cast<float4*>(scratch + kStatusBytes),
                            reinterpret_cast<float4*>(scratch + kStatusBytes + halves_bytes), rows};
    cudaError_t e = cudaMemsetAsync(ctx.status, 0, sizeof(int32_t), ctx.stream);
    if (e != cudaSuccess) return TF_ERR_CUDA;
    e = dims->dtype == TF_BF16
            ? launch_lmhead_tc(ctx, w->lm_head, hidden, rows, dims->d, dims->V, inv_temp, partials)
            : launch_lmhead_simt(ctx, dims->dtype, w->lm_head, hidden, rows, dims->d, dims->V, inv_temp, partials);
    if (e != cudaSuccess) return TF_ERR_CUDA;
    e = launch_lmhead_merge(ctx, dims->dtype, partials, rows, dims->V, dims->d, K1, inv_temp, w->lm_head, hidden,
                            top_ids, top_logp);
    if (e != cudaSuccess) return TF_ERR_CUDA;
    return from_cuda(cudaMemcpyAsync(dev_status, ctx.status, sizeof(int32_t), cudaMemcpyDeviceToDevice, ctx.stream));
}
