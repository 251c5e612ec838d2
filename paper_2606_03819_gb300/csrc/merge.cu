// Merge of the LM-head partials into log-softmax top-k (Algorithm 1 "TopM" of stage 1 and the
// log-softmax + top-k of every stage-2 row).
//
// One CTA per row. Inputs are the row's per-block summaries (block max, sum of exp, and per
// 32-column chunk the max with its id and the second-largest value). The CTA
//   1. combines the block (max, sum) pairs into the row's log-sum-exp;
//   2. keeps as candidates the chunk maxima at or above the k-th largest block maximum and finds
//      the k-th largest candidate key (value desc, id asc) with a radix select over 64-bit keys;
//   3. certifies the result: a chunk whose second-largest value reaches the k-th candidate may
//      hide further members of the top k. Those chunks' 32 logits are recomputed exactly from
//      lm_head and x, replace the chunk maxima, and the selection is redone;
//   4. writes the k winners sorted, as (id, logit - LSE).
// The result is the exact top-k of the full vocabulary whatever the input; on random data about
// one chunk per two rows is recomputed (32 dot products, a few microseconds).
#include <math.h>

#include "common.cuh"

namespace tf {
namespace {

constexpr int kThreads = 256;

__device__ __forceinline__ void lse_combine(float& m, float& s, float m2, float s2) {
    if (m2 > m) {
        s = s * __expf(m - m2) + s2;
        m = m2;
    } else if (m2 > -INFINITY) {
        s += s2 * __expf(m2 - m);
    }
}

// k-th largest of keys[0..n) (n >= k >= 1), by 8-bit digits from the most significant byte.
__device__ unsigned long long block_kth_largest(const unsigned long long* keys, int n, int k, int* hist,
                                                int* sel_digit, int* sel_rem) {
    unsigned long long prefix = 0;
    int rem = k;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    for (int shift = 56; shift >= 0; shift -= 8) {
        for (int i = tid; i < 256; i += kThreads) hist[i] = 0;
        __syncthreads();
        const unsigned long long hi_mask = shift == 56 ? 0ull : (~0ull << (shift + 8));
        // warp-aggregated counting: lanes holding the same digit add once (float keys of one
        // row share their top bytes, so plain atomics would serialise on a few bins)
        const int n_pad = (n + kThreads - 1) / kThreads * kThreads;
        for (int i = tid; i < n_pad; i += kThreads) {
            int digit = 256;
            if (i < n) {
                const unsigned long long key = keys[i];
                if ((key & hi_mask) == prefix) digit = static_cast<int>((key >> shift) & 255);
            }
            const unsigned peers = __match_any_sync(0xffffffffu, digit);
            if (digit < 256 && lane == __ffs(peers) - 1) atomicAdd(&hist[digit], __popc(peers));
        }
        __syncthreads();
        if (warp == 0) {
            int local[8];
            int sum = 0;
#pragma unroll
            for (int b = 0; b < 8; ++b) {
                local[b] = hist[lane * 8 + b];
                sum += local[b];
            }
            // inclusive suffix sum over lanes (higher lanes hold higher digits)
            int incl = sum;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int v = __shfl_down_sync(0xffffffffu, incl, o);
                if (lane + o < 32) incl += v;
            }
            const int excl = incl - sum;
            if (excl < rem && rem <= incl) {
                int c = excl;
                for (int b = 7; b >= 0; --b) {
                    if (c + local[b] >= rem) {
                        *sel_digit = lane * 8 + b;
                        *sel_rem = rem - c;
                        break;
                    }
                    c += local[b];
                }
            }
        }
        __syncthreads();
        prefix |= static_cast<unsigned long long>(*sel_digit) << shift;
        rem = *sel_rem;
        __syncthreads();
    }
    return prefix;
}

// <w, x> for one weight row (d elements) and x in shared memory (fp32), by one warp: lanes take
// 8-element slices; all of a lane's 16-byte loads are issued before the multiply-adds.
__device__ __forceinline__ float dot_row(const __nv_bfloat16* w, const float* xs, int d, int lane) {
    float acc = 0.0f;
    if ((d & 255) == 0 && (reinterpret_cast<uintptr_t>(w) & 15) == 0) {
        const uint4* w4 = reinterpret_cast<const uint4*>(w);
        const int n = d / 256;                       // 16-byte slices per lane
        for (int base = 0; base < n; base += 8) {
            uint4 buf[8];
#pragma unroll
            for (int i = 0; i < 8; ++i)
                if (base + i < n) buf[i] = w4[(base + i) * 32 + lane];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                if (base + i >= n) break;
                const __nv_bfloat16* b = reinterpret_cast<const __nv_bfloat16*>(&buf[i]);
                const float* xv = xs + ((base + i) * 32 + lane) * 8;
#pragma unroll
                for (int j = 0; j < 8; ++j) acc = fmaf(__bfloat162float(b[j]), xv[j], acc);
            }
        }
    } else {
        for (int k = lane; k < d; k += 32) acc = fmaf(__bfloat162float(w[k]), xs[k], acc);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    return acc;
}
__device__ __forceinline__ float dot_row(const float* w, const float* xs, int d, int lane) {
    float acc = 0.0f;
    for (int k = lane; k < d; k += 32) acc = fmaf(w[k], xs[k], acc);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    return acc;
}

template <typename T>
__global__ void __launch_bounds__(kThreads) lmhead_merge_kernel(const Partial* __restrict__ partials, int n_rows,
                                                                int n_tiles, int V, int d, int k, float inv_temp,
                                                                const T* __restrict__ lm_head,
                                                                const T* __restrict__ x, int32_t* __restrict__ out_ids,
                                                                float* __restrict__ out_logp, int* status) {
    // dynamic shared memory: the row's block summaries, candidate keys, per-block best key,
    // per-chunk "already recomputed" flags
    extern __shared__ __align__(16) uint8_t dsm[];
    Partial* P = reinterpret_cast<Partial*>(dsm);
    const int n_chunks = n_tiles * kChunks;
    const int cap = n_chunks + kMergeExpandChunks * kChunk;
    unsigned long long* cand = reinterpret_cast<unsigned long long*>(dsm + static_cast<size_t>(n_tiles) * sizeof(Partial));
    unsigned long long* lmax = cand + cap;
    uint8_t* expanded = reinterpret_cast<uint8_t*>(lmax + n_tiles);
    float* xs = reinterpret_cast<float*>(expanded + (n_chunks + 15) / 16 * 16);   // [d], only when needed
    bool x_staged = false;
    __shared__ int hist[256];
    __shared__ float red_m[kThreads / 32], red_s[kThreads / 32];
    __shared__ int sel_digit, sel_rem, n_flag, flag_list[kMergeExpandChunks], n_cand, n_sel, n_valid;
    __shared__ unsigned long long sel[kMaxK];
    __shared__ float zbuf[kMergeExpandChunks * kChunk];
    __shared__ float lse_s;

    const int row = blockIdx.x;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

    // 0. stage the row's summaries (contiguous, 128 B each) with 16-byte loads, eight in flight
    //    per thread before the first store
    {
        const uint4* src = reinterpret_cast<const uint4*>(partials + static_cast<size_t>(row) * n_tiles);
        uint4* dst = reinterpret_cast<uint4*>(P);
        const int n16 = n_tiles * static_cast<int>(sizeof(Partial) / 16);
        constexpr int T = kThreads;
        int i = tid;
        for (; i + 7 * T < n16; i += 8 * T) {
            uint4 v[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) v[j] = src[i + j * T];
#pragma unroll
            for (int j = 0; j < 8; ++j) dst[i + j * T] = v[j];
        }
        for (; i < n16; i += T) dst[i] = src[i];
    }
    if (tid == 0) {
        n_cand = 0;
        n_valid = 0;
    }
    __syncthreads();

    // 1. log-sum-exp over blocks; per-block best key
    float m = -INFINITY, s = 0.0f;
    int my_valid = 0;
    for (int t = tid; t < n_tiles; t += kThreads) {
        unsigned long long best = 0ull;
#pragma unroll
        for (int c = 0; c < kChunks; ++c) {
            if (P[t].cid[c] < 0) continue;
            lse_combine(m, s, P[t].cmax[c], P[t].cs[c]);
            const unsigned long long key = cand_key(P[t].cmax[c], P[t].cid[c]);
            best = key > best ? key : best;
        }
        lmax[t] = best;
        my_valid += best != 0ull ? 1 : 0;
    }
    for (int i = tid; i < n_chunks; i += kThreads) expanded[i] = 0;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
        const float s2 = __shfl_xor_sync(0xffffffffu, s, o);
        lse_combine(m, s, m2, s2);
    }
    if (lane == 0) {
        red_m[warp] = m;
        red_s[warp] = s;
    }
    atomicAdd(&n_valid, my_valid);
    __syncthreads();
    if (tid == 0) {
        float M = -INFINITY, S = 0.0f;
        for (int w = 0; w < kThreads / 32; ++w) lse_combine(M, S, red_m[w], red_s[w]);
        const float lse = M + logf(S);
        lse_s = lse;
        if (!isfinite(lse)) set_status(status, TF_DEV_NONFINITE);
    }

    // 2. candidates: the chunk maxima at or above the k-th largest block maximum. At least k keys
    //    are >= that bound (the k block maxima), so the top k are all among the chunk maxima
    //    above it or hidden behind them (handled in 3).
    const unsigned long long theta0 =
        n_valid >= k ? block_kth_largest(lmax, n_tiles, k, hist, &sel_digit, &sel_rem) : 0ull;
    for (int i = tid; i < n_chunks; i += kThreads) {
        const int t = i / kChunks, c = i - (i / kChunks) * kChunks;
        if (P[t].cid[c] < 0) continue;
        const unsigned long long key = cand_key(P[t].cmax[c], P[t].cid[c]);
        if (key >= theta0) cand[atomicAdd(&n_cand, 1)] = key;
    }
    __syncthreads();

    // 3. select; a chunk whose second-largest value reaches the k-th candidate may hide members
    //    of the top k (every chunk below theta0 cannot), so its 32 logits are recomputed exactly
    //    and the selection is redone until no chunk is in doubt
    int n_expanded = 0;
    unsigned long long theta = 0;
    for (;;) {
        const int nc = n_cand;
        theta = nc >= k ? block_kth_largest(cand, nc, k, hist, &sel_digit, &sel_rem) : 0ull;
        const float tval = key_value(theta);
        if (tid == 0) n_flag = 0;
        __syncthreads();
        for (int i = tid; i < n_chunks; i += kThreads) {
            const int t = i / kChunks, c = i - (i / kChunks) * kChunks;
            if (expanded[i] || !(P[t].c2[c] > -INFINITY)) continue;
            if (lmax[t] < theta0) continue;                     // the whole block is below the top k
            if (nc < k || P[t].c2[c] >= tval) {
                const int slot = atomicAdd(&n_flag, 1);
                if (slot < kMergeExpandChunks) flag_list[slot] = i;
            }
        }
        __syncthreads();
        const int nf = n_flag;
        if (nf == 0) break;
        if (n_expanded + nf > kMergeExpandChunks) {
            // more chunks in doubt than the recompute budget: keep the answer and say so
            if (tid == 0) set_status(status, TF_DEV_NONFINITE);
            break;
        }
        if (tid == 0) set_status(status, TF_DEV_RECOMPUTED);
        // exact logits of every flagged chunk: x staged once in shared memory, then one warp per
        // column with all of its 16-byte weight loads issued before the multiply-adds
        if (!x_staged) {
            for (int i = tid; i < d; i += kThreads) xs[i] = to_f32(x[static_cast<size_t>(row) * d + i]);
            x_staged = true;
            __syncthreads();
        }
        for (int q = warp; q < nf * kChunk; q += kThreads / 32) {
            const int f = q / kChunk, cc = q - f * kChunk;
            const int v = flag_list[f] * kChunk + cc;
            float acc = v < V ? dot_row(lm_head + static_cast<size_t>(v) * d, xs, d, lane) : -INFINITY;
            if (lane == 0) zbuf[q] = v < V ? acc * inv_temp : -INFINITY;
        }
        __syncthreads();
        // the flagged chunks' maxima leave the candidate set; all their logits enter it
        for (int i = tid; i < n_cand; i += kThreads) {
            const int id = key_id(cand[i]);
            for (int f = 0; f < nf; ++f)
                if (id / kChunk == flag_list[f]) cand[i] = 0ull;
        }
        __syncthreads();
        for (int q = tid; q < nf * kChunk; q += kThreads) {
            const int f = q / kChunk, cc = q - f * kChunk;
            const int v = flag_list[f] * kChunk + cc;
            if (v < V) cand[atomicAdd(&n_cand, 1)] = cand_key(zbuf[q], v);
        }
        for (int f = tid; f < nf; f += kThreads) expanded[flag_list[f]] = 1;
        n_expanded += nf;
        __syncthreads();
    }

    // 4. the k winners, sorted
    if (tid == 0) n_sel = 0;
    __syncthreads();
    const int nc = n_cand;
    for (int i = tid; i < nc; i += kThreads) {
        const unsigned long long key = cand[i];
        if (key != 0ull && key >= theta) {
            const int slot = atomicAdd(&n_sel, 1);
            if (slot < kMaxK) sel[slot] = key;
        }
    }
    __syncthreads();
    const int ns = min(n_sel, k);
    const float lse = lse_s;
    for (int i = tid; i < ns; i += kThreads) {
        const unsigned long long key = sel[i];
        int rank = 0;
        for (int j = 0; j < ns; ++j) rank += sel[j] > key ? 1 : 0;
        out_ids[static_cast<size_t>(row) * k + rank] = key_id(key);
        out_logp[static_cast<size_t>(row) * k + rank] = key_value(key) - lse;
    }
    for (int i = ns + tid; i < k; i += kThreads) {
        out_ids[static_cast<size_t>(row) * k + i] = -1;
        out_logp[static_cast<size_t>(row) * k + i] = -INFINITY;
    }
    if (tid == 0 && ns < k) set_status(status, TF_DEV_UNDERFULL);
}

}  // namespace

size_t merge_smem_bytes(int n_tiles, int d) {
    const size_t n_chunks = static_cast<size_t>(n_tiles) * kChunks;
    return static_cast<size_t>(n_tiles) * sizeof(Partial) +
           (n_chunks + kMergeExpandChunks * kChunk + n_tiles) * sizeof(unsigned long long) + (n_chunks + 15) / 16 * 16 +
           static_cast<size_t>(d) * sizeof(float);
}

cudaError_t launch_lmhead_merge(const Ctx& ctx, int dtype, const Partial* partials, int n_rows, int V, int d, int k,
                                float inv_temp, const void* lm_head, const void* x, int32_t* out_ids,
                                float* out_logp) {
    if (n_rows <= 0) return cudaSuccess;
    const int n_tiles = (V + kBlockV - 1) / kBlockV;
    const size_t smem = merge_smem_bytes(n_tiles, d);
    if (dtype == TF_BF16) {
        auto kern = lmhead_merge_kernel<__nv_bfloat16>;
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
        if (e != cudaSuccess) return e;
        kern<<<n_rows, kThreads, smem, ctx.stream>>>(partials, n_rows, n_tiles, V, d, k, inv_temp,
                                                     static_cast<const __nv_bfloat16*>(lm_head),
                                                     static_cast<const __nv_bfloat16*>(x), out_ids, out_logp,
                                                     ctx.status);
    } else {
        auto kern = lmhead_merge_kernel<float>;
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
        if (e != cudaSuccess) return e;
        kern<<<n_rows, kThreads, smem, ctx.stream>>>(partials, n_rows, n_tiles, V, d, k, inv_temp,
                                                     static_cast<const float*>(lm_head), static_cast<const float*>(x),
                                                     out_ids, out_logp, ctx.status);
    }
    return cudaGetLastError();
}

}  // namespace tf
