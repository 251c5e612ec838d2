// Split-K reductions of the approximator GEMMs (Eq. 1). The tensor-core kernels leave fp32
// partial sums [k_splits][N / 4][rows][4]; these kernels add them in a fixed order and apply the rest
// of the layer: SiLU(G) * U for the gate/up GEMM, the residual h for the down GEMM. Outputs are
// bf16, rounded once, exactly as the unsplit epilogues do.
#include <math.h>

#include "common.cuh"

namespace tf {
namespace {

__device__ __forceinline__ float4 add4(float4 a, float4 b) {
    return make_float4(a.x + b.x, a.y + b.y, a.z + b.z, a.w + b.w);
}
__device__ __forceinline__ float silu_f(float g) { return g / (1.0f + __expf(-g)); }

// The partial tables are float4-major, [ks][columns / 4][rows][4] (what the tensor-core
// epilogue stores): thread idx takes the four columns 4 (idx / rows) .. + 3 of row idx % rows,
// so a warp reads 512 contiguous bytes per split.

// partial [ks][2I / 4][rows][4] (gate in columns [0, I), up in [I, 2I)) -> A [rows][I]
__global__ void __launch_bounds__(256) swiglu_reduce_kernel(const float4* __restrict__ partial, int ks, int rows,
                                                            int I, __nv_bfloat162* __restrict__ A) {
    pdl_trigger();
    pdl_wait();
    const size_t n = static_cast<size_t>(I / 4) * rows;
    const size_t split = 2 * n;   // float4s per k split
    for (size_t idx = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; idx < n;
         idx += static_cast<size_t>(gridDim.x) * blockDim.x) {
        const int r = static_cast<int>(idx % rows);
        const size_t c4 = idx / rows;   // column group: columns 4 c4 .. 4 c4 + 3
        const float4* p = partial + idx;   // gate; up is I / 4 column groups later
        float4 g = p[0], u = p[n];
        for (int k = 1; k < ks; ++k) {
            g = add4(g, p[k * split]);
            u = add4(u, p[k * split + n]);
        }
        __nv_bfloat162* dst = A + (static_cast<size_t>(r) * I + c4 * 4) / 2;
        dst[0] = __floats2bfloat162_rn(silu_f(g.x) * u.x, silu_f(g.y) * u.y);
        dst[1] = __floats2bfloat162_rn(silu_f(g.z) * u.z, silu_f(g.w) * u.w);
    }
}

// partial [ks][d / 4][rows][4] -> h' [rows][d] = h[stage-2 row's hidden state] + sum
__global__ void __launch_bounds__(256) down_reduce_kernel(const float4* __restrict__ partial, int ks, int rows, int d,
                                                          const __nv_bfloat162* __restrict__ hidden, int R, int M,
                                                          int gamma, __nv_bfloat162* __restrict__ hp) {
    pdl_trigger();
    pdl_wait();
    const size_t n = static_cast<size_t>(d / 4) * rows;
    for (size_t idx = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; idx < n;
         idx += static_cast<size_t>(gridDim.x) * blockDim.x) {
        const int r = static_cast<int>(idx % rows);
        const size_t c4 = idx / rows;
        float4 a = partial[idx];
        for (int k = 1; k < ks; ++k) a = add4(a, partial[k * n + idx]);
        const int sq = r / R, rr = r - sq * R;
        const size_t hrow = static_cast<size_t>(sq) * gamma + stage2_hidden_index(rr, M);
        const size_t col2 = c4 * 2;
        const __nv_bfloat162 h0 = hidden[hrow * (d / 2) + col2], h1 = hidden[hrow * (d / 2) + col2 + 1];
        __nv_bfloat162* dst = hp + static_cast<size_t>(r) * (d / 2) + col2;
        dst[0] = __floats2bfloat162_rn(__bfloat162float(h0.x) + a.x, __bfloat162float(h0.y) + a.y);
        dst[1] = __floats2bfloat162_rn(__bfloat162float(h1.x) + a.z, __bfloat162float(h1.y) + a.w);
    }
}

int grid_for(size_t n, const Ctx& ctx) {
    const size_t want = (n + 255) / 256;
    const size_t cap = static_cast<size_t>(ctx.num_sms) * 8;
    return static_cast<int>(want < cap ? want : cap);
}

}  // namespace

cudaError_t launch_swiglu_reduce(const Ctx& ctx, const float* partial, int k_splits, int n_rows, int I,
                                 __nv_bfloat16* A) {
    const size_t n = static_cast<size_t>(n_rows) * (I / 4);
    const cudaError_t e = launch_pdl(swiglu_reduce_kernel, dim3(grid_for(n, ctx)), dim3(256), 0, ctx.stream,
                                     reinterpret_cast<const float4*>(partial), k_splits, n_rows, I,
                                     reinterpret_cast<__nv_bfloat162*>(A));
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t launch_down_reduce(const Ctx& ctx, const float* partial, int k_splits, int n_rows, int d,
                               const __nv_bfloat16* hidden, int R, int M, int gamma, __nv_bfloat16* h_prime) {
    const size_t n = static_cast<size_t>(n_rows) * (d / 4);
    const cudaError_t e = launch_pdl(down_reduce_kernel, dim3(grid_for(n, ctx)), dim3(256), 0, ctx.stream,
                                     reinterpret_cast<const float4*>(partial), k_splits, n_rows, d,
                                     reinterpret_cast<const __nv_bfloat162*>(hidden), R, M, gamma,
                                     reinterpret_cast<__nv_bfloat162*>(h_prime));
    return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace tf
