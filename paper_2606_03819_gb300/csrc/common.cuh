// Shared definitions of the TreeFlash CUDA library (device side and launcher side).
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "treeflash.h"

namespace tf {

// ---- sizes fixed by the kernels --------------------------------------------------------------
constexpr int kBlockV = 256;        // vocabulary entries per LM-head block (one MMA N-tile)
constexpr int kChunk = 32;           // vocabulary columns per chunk (one TMEM load per row)
constexpr int kChunks = kBlockV / kChunk;  // chunks per block
constexpr int kMaxK = 512;          // largest top-k a merge can return
constexpr int kMaxM = 64;           // largest M (the builder tests membership with two ballots)
constexpr int kMaxB = 1023;         // largest draft budget
constexpr int kMaxGamma = 64;
constexpr int kMergeExpandChunks = 64;     // chunks a merge may recompute exactly
constexpr int kMaxKSplits = 4;        // split-K factor of the approximator GEMMs (workspace sized for it)
// Counters of the approximator GEMMs' tail split (K-chunks of the units of a last, partial round),
// kept in the workspace right after the status word and zeroed by the gather of every call.
constexpr int kTailSems = 1024;
constexpr int kMaxTailSplit = 8;       // K-chunks per tail unit

// What the LM-head pass leaves per (row, vocabulary block of 256). Both arrays are indexed
// [block][part][row], so the 32 lanes of an epilogue warp (32 consecutive rows) store 512
// contiguous bytes per record.
//  - halves [n_tiles][2][n_rows]: per half block (128 columns = 4 chunks) the max logit m, the
//    sum over the half of exp(z - m), and the half's best (value, id bits). The merge reads only
//    these for the log-sum-exp and its first threshold.
//  - chunks [n_tiles][kChunks][n_rows]: per 32-column chunk its largest, second and third largest
//    logits and, in .w, the chunk-local offsets of the first two (bits 0-7 and 8-15). Read only
//    for the halves that can hold members of the top k: the two largest are candidates, the third
//    bounds every other logit of the chunk.
// Ties go to the smaller id. Empty entries have -inf values and sum 0.
struct Partials {
    float4* halves;
    float4* chunks;
    int n_rows;
    __host__ __device__ size_t half_at(int tile, int half, int row) const {
        return (static_cast<size_t>(tile) * 2 + half) * n_rows + row;
    }
    __host__ __device__ size_t chunk_at(int tile, int chunk, int row) const {
        return (static_cast<size_t>(tile) * kChunks + chunk) * n_rows + row;
    }
};
constexpr size_t kHalfBytesPerRowBlock = 2 * sizeof(float4);
constexpr size_t kChunkBytesPerRowBlock = kChunks * sizeof(float4);

// ---- bf16 / f32 element access ----------------------------------------------------------------
__device__ __forceinline__ float to_f32(float x) { return x; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 x) { return __bfloat162float(x); }
template <typename T> __device__ __forceinline__ T from_f32(float x);
template <> __device__ __forceinline__ float from_f32<float>(float x) { return x; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float x) {
    return __float2bfloat16_rn(x);
}

// Order-preserving map of a float to uint32 (larger float -> larger key; -0 < +0; NaN ends up
// above +inf or below -inf depending on its sign bit, it never appears in practice).
__device__ __forceinline__ uint32_t float_key(float f) {
    uint32_t u = __float_as_uint(f);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float key_float(uint32_t k) {
    uint32_t u = (k & 0x80000000u) ? (k & 0x7fffffffu) : ~k;
    return __uint_as_float(u);
}
// 64-bit candidate key: larger value first, then smaller token id.
__device__ __forceinline__ unsigned long long cand_key(float v, int id) {
    return ((unsigned long long)float_key(v) << 32) | (unsigned long long)(0xffffffffu - (uint32_t)id);
}
__device__ __forceinline__ int key_id(unsigned long long k) {
    return (int)(0xffffffffu - (uint32_t)(k & 0xffffffffull));
}
__device__ __forceinline__ float key_value(unsigned long long k) { return key_float((uint32_t)(k >> 32)); }

__device__ __forceinline__ void set_status(int* status, int bits) {
    if (status) atomicOr(status, bits);
}

// Stage-2 row -> (index of the hidden state it refines within its sequence, previous-token
// source). Row 0 of a sequence refines h_{t+1} with the root token; row 1 + (i-2) M + m
// refines h_{t+i} with stage-1 candidate m of depth i-1 (Algorithm 1 Part 1, 1 + M(gamma-1)
// rows per sequence).
__host__ __device__ __forceinline__ int stage2_hidden_index(int r, int M) {
    return r == 0 ? 0 : (r - 1) / M + 1;
}

// ---- programmatic dependent launch ---------------------------------------------------------
// Every kernel of the path is launched so that it may start while the previous kernel on the
// stream is finishing. pdl_wait() blocks until the previous kernel has completed and its writes
// are visible; each kernel calls it, on every path, before it reads anything an earlier kernel
// wrote or writes anything an earlier kernel may still read. Only reads of the weights (which
// no kernel writes) and on-chip set-up come before it. pdl_trigger() lets the next kernel be
// scheduled; where it is called only decides how early the next kernel's set-up may overlap.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" :::); }

// Host-side count of kernels launched by this library (tf_kernel_launches).
void note_launch();
// Limit of the tensor-core kernels' waits for progress, set by tf_set_wait_limit_ns (0: the
// kernels' own default).
unsigned long long wait_limit_ns();

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                       Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const cudaError_t e = cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
    if (e == cudaSuccess) note_launch();
    return e;
}

// The same launch with thread-block clusters of cluster_x CTAs along x.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl_cluster(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                               int cluster_x, Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = cluster_x;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    const cudaError_t e = cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
    if (e == cudaSuccess) note_launch();
    return e;
}

}  // namespace tf

// ---- launchers (one per kernel family); implemented in the .cu files -------------------------
namespace tf {

struct Ctx {
    cudaStream_t stream;
    int num_sms;
    int* status;  // device status word in the workspace
};

// LM-head pass (tensor-core path for bf16, CUDA-core path for f32); reset_status: the kernel
// zeroes ctx.status once every earlier kernel on the stream has finished
cudaError_t launch_lmhead_tc(const Ctx&, const void* lm_head, const void* x, int n_rows, int d,
                             int V, float inv_temp, Partials partials, bool reset_status = false);
cudaError_t launch_lmhead_simt(const Ctx&, int dtype, const void* lm_head, const void* x,
                               int n_rows, int d, int V, float inv_temp, Partials partials,
                               bool reset_status = false);
cudaError_t launch_lmhead_merge(const Ctx&, int dtype, Partials partials, int n_rows, int V,
                                int d, int k, float inv_temp, const void* lm_head, const void* x,
                                int32_t* out_ids, float* out_logp);
// Eq. 1 pieces
// x rows of stage 2 (R per sequence). two_prev: x = [h~ ; e(prev) ; e(token before prev)] (3d
// wide) and root_tok holds two tokens per sequence; hres (two_prev only) receives each row's
// residual hidden state.
cudaError_t launch_gather_norm(const Ctx&, int dtype, const void* hidden, const void* embed,
                               const void* norm_h, const void* norm_e, const int32_t* root_tok,
                               const int32_t* top_ids, int b, int gamma, int M, int K1, int R,
                               int two_prev, int d, int V, float eps, void* X, void* hres);
// SwiGLU on x [n_rows, k_in] (k_in = 2d, or 3d with two previous tokens)
cudaError_t launch_swiglu_tc(const Ctx&, const void* X, int k_in, const void* w_gate,
                             const void* w_up, const void* w_down, const void* hidden, int n_rows,
                             int d, int I, int R, int M, int gamma, void* A, void* h_prime,
                             float* partial, size_t partial_bytes);
// bytes of the split-K exchange area of the cluster path for a GEMM with n_out_cols output columns
// made of nb adjacent matrices (the workspace's partial-sum region must hold it)
size_t splitk_exchange_bytes(int n_out_cols, int nb);
// split-K reductions of the approximator GEMMs (partial sums in fp32, [k_splits][N / 4][rows][4])
cudaError_t launch_swiglu_reduce(const Ctx&, const float* partial, int k_splits, int n_rows, int I,
                                 __nv_bfloat16* A);
cudaError_t launch_down_reduce(const Ctx&, const float* partial, int k_splits, int n_rows, int d,
                               const __nv_bfloat16* hidden, int R, int M, int gamma,
                               __nv_bfloat16* h_prime);
cudaError_t launch_swiglu_simt(const Ctx&, const void* X, int k_in, const void* w_gate,
                               const void* w_up, const void* w_down, const void* hidden,
                               int n_rows, int d, int I, int R, int M, int gamma, void* A,
                               void* h_prime);
// the "w/ Linear" approximator: h' = h + X W_lin^T, X [n_rows, 2d], W_lin [d, 2d]
cudaError_t launch_linear_tc(const Ctx&, const void* X, const void* w_lin, const void* hidden,
                             int n_rows, int d, int R, int M, int gamma, void* h_prime,
                             float* partial, size_t partial_bytes);
cudaError_t launch_linear_simt(const Ctx&, const void* X, const void* w_lin, const void* hidden,
                               int n_rows, int d, int R, int M, int gamma, void* h_prime);
// Part 2 and the mask
cudaError_t launch_build_tree(const Ctx&, int b, int gamma, int M, int K1, int K2, int B, int V,
                              int mode, int R, int two_prev, const int32_t* root_tok,
                              const int32_t* top_ids,
                              const float* top_logp, const int32_t* child_ids,
                              const float* child_logp, int32_t* node_tok, int32_t* node_parent,
                              int32_t* node_depth, float* node_score, int32_t* dev_status,
                              const int32_t* root_pos = nullptr, uint8_t* mask = nullptr,
                              int32_t* pos_ids = nullptr, const int32_t* ws_status = nullptr);
// the largest tree (B + 1 nodes) whose mask launch_build_tree can write from the builder itself
constexpr int kFusedMaskMaxNodes = 128;
cudaError_t launch_accept_walk(const Ctx&, int b, int B, int gamma, const int32_t* node_tok,
                               const int32_t* node_parent, const int32_t* verifier_tok,
                               int32_t* accept_len, int32_t* accept_path, int32_t* next_tok);
cudaError_t launch_tree_mask(const Ctx&, int b, int B, const int32_t* node_parent,
                             const int32_t* node_depth, const int32_t* root_pos, uint8_t* mask,
                             int32_t* pos_ids);

}  // namespace tf
