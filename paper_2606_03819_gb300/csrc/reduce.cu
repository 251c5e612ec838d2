// Split-K reductions of the approximator GEMMs (Eq. 1). The tensor-core kernels leave fp32
// partial sums [k_splits][rows][N]; these kernels add them in a fixed order and apply the rest
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

// partial [ks][rows][2I] (gate in columns [0, I), up in [I, 2I)) -> A [rows][I]
__global__ void __launch_bounds__(256) swiglu_reduce_kernel(const float4* __restrict__ partial, int ks, int rows,
                                                            int I, __nv_bfloat162* __restrict__ A) {
    pdl_trigger();
    pdl_wait();
    const int i4 = I / 4;
    const size_t n = static_cast<size_t>(rows) * i4;
    const size_t split = static_cast<size_t>(rows) * 2 * i4;
    for (size_t idx = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; idx < n;
         idx += static_cast<size_t>(gridDim.x) * blockDim.x) {
        const size_t r = idx / i4, j = idx - r * i4;
        const float4* p = partial + r * 2 * i4 + j;
        float4 g = p[0], u = p[i4];
        for (int k = 1; k < ks; ++k) {
            g = add4(g, p[k * split]);
            u = add4(u, p[k * split + i4]);
        }
        A[idx * 2] = __floats2bfloat162_rn(silu_f(g.x) * u.x, silu_f(g.y) * u.y);
        A[idx * 2 + 1] = __floats2bfloat162_rn(silu_f(g.z) * u.z, silu_f(g.w) * u.w);
    }
}

// partial [ks][rows][d] -> h' [rows][d] = h[stage-2 row's hidden state] + sum
__global__ void __launch_bounds__(256) down_reduce_kernel(const float4* __restrict__ partial, int ks, int rows, int d,
                                                          const __nv_bfloat162* __restrict__ hidden, int R, int M,
                                                          int gamma, __nv_bfloat162* __restrict__ hp) {
    pdl_trigger();
    pdl_wait();
    const int d4 = d / 4;
    const size_t n = static_cast<size_t>(rows) * d4;
    const size_t split = n;
    for (size_t idx = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; idx < n;
         idx += static_cast<size_t>(gridDim.x) * blockDim.x) {
        const int r = static_cast<int>(idx / d4);
        const size_t c = idx - static_cast<size_t>(r) * d4;
        float4 a = partial[idx];
        for (int k = 1; k < ks; ++k) a = add4(a, partial[k * split + idx]);
        const int sq = r / R, rr = r - sq * R;
        const size_t hrow = static_cast<size_t>(sq) * gamma + stage2_hidden_index(rr, M);
        const __nv_bfloat162 h0 = hidden[(hrow * d4 + c) * 2], h1 = hidden[(hrow * d4 + c) * 2 + 1];
        hp[idx * 2] = __floats2bfloat162_rn(__bfloat162float(h0.x) + a.x, __bfloat162float(h0.y) + a.y);
        hp[idx * 2 + 1] = __floats2bfloat162_rn(__bfloat162float(h1.x) + a.z, __bfloat162float(h1.y) + a.w);
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
