// CUDA-core (fp32 FMA) kernels of the TF_F32 path: the same LM-head pass and SwiGLU of Eq. 1
// as the tensor-core path, for fp32 inputs whose 1e-4 accuracy target rules out TF32 / bf16
// tensor-core arithmetic. Same partial format, same merge.
#include <math.h>

#include "common.cuh"

namespace tf {
namespace {

constexpr int kRowsPerCta = 32;
constexpr int kKChunk = 32;

// One CTA: rows [r0, r0 + 32) x vocabulary block [v0, v0 + 256). Thread t owns vocabulary column
// v0 + t and accumulates its 32 logits; the block is then staged in shared memory and one warp
// per row computes, with warp shuffles, the per-chunk three largest logits (ids of the first
// two) and the per-half max, sum of exp and best entry.
__global__ void __launch_bounds__(256) lmhead_simt_kernel(const float* __restrict__ W, const float* __restrict__ X,
                                                          int n_rows, int d, int V, float inv_temp,
                                                          Partials partials, int n_tiles, int* reset_status) {
    pdl_trigger();
    pdl_wait();
    if (reset_status && blockIdx.x == 0 && blockIdx.y == 0 && threadIdx.x == 0) *reset_status = 0;
    __shared__ float xs[kRowsPerCta][kKChunk + 1];
    __shared__ float ws[kBlockV][kKChunk + 1];
    const int vt = blockIdx.x;
    const int r0 = blockIdx.y * kRowsPerCta;
    const int t = threadIdx.x;
    float acc[kRowsPerCta];
#pragma unroll
    for (int r = 0; r < kRowsPerCta; ++r) acc[r] = 0.0f;

    for (int k0 = 0; k0 < d; k0 += kKChunk) {
        for (int i = t; i < kRowsPerCta * kKChunk; i += 256) {
            const int r = i / kKChunk, k = i % kKChunk;
            xs[r][k] = (r0 + r < n_rows && k0 + k < d) ? X[static_cast<size_t>(r0 + r) * d + k0 + k] : 0.0f;
        }
        for (int i = t; i < kBlockV * kKChunk; i += 256) {
            const int v = i / kKChunk, k = i % kKChunk;
            const int gv = vt * kBlockV + v;
            ws[v][k] = (gv < V && k0 + k < d) ? W[static_cast<size_t>(gv) * d + k0 + k] : 0.0f;
        }
        __syncthreads();
#pragma unroll 4
        for (int k = 0; k < kKChunk; ++k) {
            const float w = ws[t][k];
#pragma unroll
            for (int r = 0; r < kRowsPerCta; ++r) acc[r] = fmaf(xs[r][k], w, acc[r]);
        }
        __syncthreads();
    }
    // stage the logits of the block: zt[r][t]
    float* zt = &ws[0][0];
    const bool valid = vt * kBlockV + t < V;
#pragma unroll
    for (int r = 0; r < kRowsPerCta; ++r) zt[r * kBlockV + t] = valid ? acc[r] * inv_temp : -INFINITY;
    __syncthreads();

    const int warp = t >> 5, lane = t & 31;
    for (int r = warp; r < kRowsPerCta; r += 8) {
        if (r0 + r >= n_rows) break;
        // chunk j = columns [32 j, 32 j + 32) of the block; lane holds column 32 j + lane
        float z[kChunks];
#pragma unroll
        for (int j = 0; j < kChunks; ++j) z[j] = zt[r * kBlockV + lane + 32 * j];
        const int row = r0 + r;
        float hm[2] = {-INFINITY, -INFINITY}, hsum[2] = {0.0f, 0.0f}, hbv[2] = {-INFINITY, -INFINITY};
        int hbid[2] = {-1, -1};
#pragma unroll
        for (int j = 0; j < kChunks; ++j) {
            const int cbase = vt * kBlockV + 32 * j;
            // three rounds of a warp-wide (value desc, id asc) arg-max over the chunk
            float x = z[j];
            float tv[3];
            int ti[3];
#pragma unroll
            for (int t3 = 0; t3 < 3; ++t3) {
                float bv = x;
                int bid = x > -INFINITY ? lane : 64;
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) {
                    const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
                    const int oid = __shfl_xor_sync(0xffffffffu, bid, o);
                    if (ov > bv || (ov == bv && oid < bid)) {
                        bv = ov;
                        bid = oid;
                    }
                }
                tv[t3] = bv;
                ti[t3] = bv > -INFINITY ? bid : 0;
                if (bv > -INFINITY && lane == bid) x = -INFINITY;
            }
            float e = tv[0] > -INFINITY ? expf(z[j] - tv[0]) : 0.0f;
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) e += __shfl_xor_sync(0xffffffffu, e, o);
            const int h = j / (kChunks / 2);
            if (tv[0] > hbv[h]) {
                hbv[h] = tv[0];
                hbid[h] = cbase + ti[0];
            }
            if (tv[0] > -INFINITY) {
                const float mn = fmaxf(hm[h], tv[0]);
                hsum[h] = hsum[h] * expf(hm[h] - mn) + e * expf(tv[0] - mn);
                hm[h] = mn;
            }
            if (lane == 0)
                partials.chunks[partials.chunk_at(vt, j, row)] =
                    make_float4(tv[0], tv[1], tv[2], __int_as_float(ti[0] | (ti[1] << 8)));
        }
        if (lane == 0)
            for (int h = 0; h < 2; ++h)
                partials.halves[partials.half_at(vt, h, row)] = make_float4(hm[h], hsum[h], hbv[h], __int_as_float(hbid[h]));
    }
}

// C[n_rows, N] = X[n_rows, K] W[N, K]^T on 64 x 64 tiles (16 x 16 threads, 4 x 4 outputs each).
// GATEUP: out = SiLU(X Wg^T) * (X Wu^T); DOWN: out = hidden[stage-2 row's depth] + X Wd^T.
template <bool GATEUP>
__global__ void __launch_bounds__(256) swiglu_simt_kernel(const float* __restrict__ X, const float* __restrict__ W0,
                                                          const float* __restrict__ W1, int n_rows, int K, int N,
                                                          float* __restrict__ out, const float* __restrict__ hidden,
                                                          int R, int M, int gamma) {
    pdl_trigger();
    pdl_wait();
    constexpr int T = 64, KC = 16;
    __shared__ float xs[KC][T + 4];
    __shared__ float w0s[KC][T + 4];
    __shared__ float w1s[GATEUP ? KC : 1][T + 4];
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    const int row0 = blockIdx.y * T, col0 = blockIdx.x * T;
    float a0[4][4] = {}, a1[4][4] = {};
    for (int k0 = 0; k0 < K; k0 += KC) {
        for (int i = threadIdx.x; i < T * KC; i += 256) {
            const int r = i / KC, k = i % KC;
            const bool kin = k0 + k < K;
            xs[k][r] = (row0 + r < n_rows && kin) ? X[static_cast<size_t>(row0 + r) * K + k0 + k] : 0.0f;
            w0s[k][r] = (col0 + r < N && kin) ? W0[static_cast<size_t>(col0 + r) * K + k0 + k] : 0.0f;
            if (GATEUP) w1s[k][r] = (col0 + r < N && kin) ? W1[static_cast<size_t>(col0 + r) * K + k0 + k] : 0.0f;
        }
        __syncthreads();
#pragma unroll
        for (int k = 0; k < KC; ++k) {
            float xv[4], wv0[4], wv1[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                xv[i] = xs[k][ty * 4 + i];
                wv0[i] = w0s[k][tx * 4 + i];
                if (GATEUP) wv1[i] = w1s[k][tx * 4 + i];
            }
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    a0[i][j] = fmaf(xv[i], wv0[j], a0[i][j]);
                    if (GATEUP) a1[i][j] = fmaf(xv[i], wv1[j], a1[i][j]);
                }
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int r = row0 + ty * 4 + i;
        if (r >= n_rows) continue;
        int hid = 0;
        if (!GATEUP) {
            const int sq = r / R, rr = r - sq * R;
            hid = sq * gamma + stage2_hidden_index(rr, M);
        }
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int c = col0 + tx * 4 + j;
            if (c >= N) continue;
            float v;
            if (GATEUP) {
                const float g = a0[i][j];
                v = g / (1.0f + expf(-g)) * a1[i][j];
            } else {
                v = hidden[static_cast<size_t>(hid) * N + c] + a0[i][j];
            }
            out[static_cast<size_t>(r) * N + c] = v;
        }
    }
}

}  // namespace

cudaError_t launch_lmhead_simt(const Ctx& ctx, int dtype, const void* lm_head, const void* x, int n_rows, int d,
                               int V, float inv_temp, Partials partials, bool reset_status) {
    if (dtype != TF_F32) return cudaErrorNotSupported;
    if (n_rows <= 0) return cudaSuccess;
    const int n_tiles = (V + kBlockV - 1) / kBlockV;
    dim3 grid(n_tiles, (n_rows + kRowsPerCta - 1) / kRowsPerCta);
    const cudaError_t e = launch_pdl(lmhead_simt_kernel, grid, dim3(256), 0, ctx.stream,
                                     static_cast<const float*>(lm_head), static_cast<const float*>(x), n_rows, d, V,
                                     inv_temp, partials, n_tiles, reset_status ? ctx.status : static_cast<int*>(nullptr));
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t launch_swiglu_simt(const Ctx& ctx, const void* X, int k_in, const void* w_gate, const void* w_up,
                               const void* w_down, const void* hidden, int n_rows, int d, int I, int R, int M,
                               int gamma, void* A, void* h_prime) {
    if (n_rows <= 0) return cudaSuccess;
    dim3 g1((I + 63) / 64, (n_rows + 63) / 64);
    cudaError_t e = launch_pdl(swiglu_simt_kernel<true>, g1, dim3(256), 0, ctx.stream, static_cast<const float*>(X),
                               static_cast<const float*>(w_gate), static_cast<const float*>(w_up), n_rows, k_in, I,
                               static_cast<float*>(A), static_cast<const float*>(nullptr), R, M, gamma);
    if (e == cudaSuccess) e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    dim3 g2((d + 63) / 64, (n_rows + 63) / 64);
    e = launch_pdl(swiglu_simt_kernel<false>, g2, dim3(256), 0, ctx.stream, static_cast<const float*>(A),
                   static_cast<const float*>(w_down), static_cast<const float*>(nullptr), n_rows, I, d,
                   static_cast<float*>(h_prime), static_cast<const float*>(hidden), R, M, gamma);
    return e != cudaSuccess ? e : cudaGetLastError();
}

// The "w/ Linear" approximator: the residual GEMM above with x (K = 2d) in place of A.
cudaError_t launch_linear_simt(const Ctx& ctx, const void* X, const void* w_lin, const void* hidden, int n_rows, int d,
                               int R, int M, int gamma, void* h_prime) {
    if (n_rows <= 0) return cudaSuccess;
    dim3 grid((d + 63) / 64, (n_rows + 63) / 64);
    const cudaError_t e = launch_pdl(swiglu_simt_kernel<false>, grid, dim3(256), 0, ctx.stream,
                                     static_cast<const float*>(X), static_cast<const float*>(w_lin),
                                     static_cast<const float*>(nullptr), n_rows, 2 * d, d,
                                     static_cast<float*>(h_prime), static_cast<const float*>(hidden), R, M, gamma);
    return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace tf
