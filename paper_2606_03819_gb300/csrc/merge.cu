// Merge of the LM-head partials into log-softmax top-k (Algorithm 1 "TopM" of stage 1 and the
// log-softmax + top-k of every stage-2 row).
//
// One CTA per row. Inputs are the row's per-block summaries (max, sum of exp, 8 largest). The
// CTA
//   1. combines the block (max, sum) pairs into the row's log-sum-exp;
//   2. keeps as candidates the entries at or above the k-th largest block maximum (at least k
//      keys lie there, so the top k do too) and finds the k-th largest candidate key (value
//      desc, id asc) with an 8-pass radix select over 64-bit keys;
//   3. certifies the result: a block whose list is full (8 entries) and whose smallest kept
//      entry still beats the k-th key may hide further members of the top-k. Such blocks
//      (at most (k-1)/8 of them, since their 8 entries all lie in the top k-1) get their 256
//      logits recomputed exactly from lm_head and x, and the selection is redone;
//   4. writes the k winners sorted, as (id, logit - LSE).
// The result is therefore the exact top-k of the full vocabulary whatever the input.
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

template <typename T>
__global__ void __launch_bounds__(kThreads) lmhead_merge_kernel(const Partial* __restrict__ partials, int n_rows,
                                                                int n_tiles, int V, int d, int k, float inv_temp,
                                                                const T* __restrict__ lm_head,
                                                                const T* __restrict__ x, int32_t* __restrict__ out_ids,
                                                                float* __restrict__ out_logp, int* status) {
    // dynamic shared memory: the row's block summaries, then candidate keys
    extern __shared__ __align__(16) uint8_t dsm[];
    Partial* P = reinterpret_cast<Partial*>(dsm);
    const int n_base = n_tiles * kListLen;
    const int cap = n_base + kMergeExpandLists * kMaxK;
    unsigned long long* cand = reinterpret_cast<unsigned long long*>(dsm + static_cast<size_t>(n_tiles) * sizeof(Partial));
    unsigned long long* lmax = cand + cap;       // per-block best key
    uint8_t* expanded = reinterpret_cast<uint8_t*>(lmax + n_tiles);
    __shared__ int hist[256];
    __shared__ float red_m[kThreads / 32], red_s[kThreads / 32];
    __shared__ int sel_digit, sel_rem, n_flag, flag_list[kMergeExpandLists + 1], n_cand, n_sel, n_valid;
    __shared__ unsigned long long sel[kMaxK];
    __shared__ float zbuf[kBlockV];
    __shared__ float lse_s;

    const int row = blockIdx.x;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

    // 0. stage the row's summaries (contiguous, 72 B = 9 x 8 B each) with 8-byte loads; a row
    //    starts on an 8-byte boundary for any n_tiles (16 only when n_tiles is even)
    {
        const uint2* src = reinterpret_cast<const uint2*>(partials + static_cast<size_t>(row) * n_tiles);
        uint2* dst = reinterpret_cast<uint2*>(P);
        const int n8 = n_tiles * static_cast<int>(sizeof(Partial) / 8);
        for (int i = tid; i < n8; i += kThreads) dst[i] = src[i];
    }
    if (tid == 0) {
        n_cand = 0;
        n_valid = 0;
    }
    __syncthreads();

    // 1. log-sum-exp over blocks
    float m = -INFINITY, s = 0.0f;
    for (int t = tid; t < n_tiles; t += kThreads) lse_combine(m, s, P[t].m, P[t].s);
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
    // per-block best keys (0 = empty block)
    int my_valid = 0;
    for (int t = tid; t < n_tiles; t += kThreads) {
        const int id = P[t].id[0];
        lmax[t] = id >= 0 ? cand_key(P[t].v[0], id) : 0ull;
        expanded[t] = 0;
        my_valid += id >= 0 ? 1 : 0;
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

    // 2. candidates: every kept entry at or above the k-th largest block maximum. At least k
    //    keys are >= that bound (the k block maxima), so the top k are all among them.
    const unsigned long long theta0 =
        n_valid >= k ? block_kth_largest(lmax, n_tiles, k, hist, &sel_digit, &sel_rem) : 0ull;
    for (int t = tid; t < n_tiles; t += kThreads) {
        for (int j = 0; j < kListLen; ++j) {
            const int id = P[t].id[j];
            if (id < 0) break;
            const unsigned long long key = cand_key(P[t].v[j], id);
            if (key < theta0) break;            // lists are sorted: the rest is smaller
            cand[atomicAdd(&n_cand, 1)] = key;
        }
    }
    __syncthreads();

    // 3. select, certify, recompute flagged blocks, repeat
    int n_expanded = 0;
    unsigned long long theta = 0;
    for (;;) {
        const int nc = n_cand;
        theta = nc >= k ? block_kth_largest(cand, nc, k, hist, &sel_digit, &sel_rem) : 0ull;
        if (tid == 0) n_flag = 0;
        __syncthreads();
        for (int t = tid; t < n_tiles; t += kThreads) {
            if (expanded[t] || P[t].id[kListLen - 1] < 0) continue;
            const unsigned long long last = cand_key(P[t].v[kListLen - 1], P[t].id[kListLen - 1]);
            if (last > theta) {
                const int slot = atomicAdd(&n_flag, 1);
                if (slot < kMergeExpandLists + 1) flag_list[slot] = t;
            }
        }
        __syncthreads();
        const int nf = n_flag;
        if (nf == 0) break;
        if (n_expanded + nf > kMergeExpandLists) {
            // cannot happen for k <= 64 (see above); keep the truncated answer and say so
            if (tid == 0) set_status(status, TF_DEV_NONFINITE);
            break;
        }
        if (tid == 0) set_status(status, TF_DEV_RECOMPUTED);
        for (int f = 0; f < nf; ++f) {
            const int t = flag_list[f];
            const int v0 = t * kBlockV;
            const int cols = min(kBlockV, V - v0);
            // exact logits of the block for this row (one warp per column, lanes split d)
            for (int c = warp; c < cols; c += kThreads / 32) {
                const T* wr = lm_head + static_cast<size_t>(v0 + c) * d;
                const T* xr = x + static_cast<size_t>(row) * d;
                float acc = 0.0f;
                for (int kk = lane; kk < d; kk += 32) acc = fmaf(to_f32(wr[kk]), to_f32(xr[kk]), acc);
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
                if (lane == 0) zbuf[c] = acc * inv_temp;
            }
            __syncthreads();
            // the block's old (truncated) entries leave the candidate set
            for (int i = tid; i < n_cand; i += kThreads) {
                const int id = key_id(cand[i]);
                if (id >= v0 && id < v0 + cols) cand[i] = 0ull;
            }
            __syncthreads();
            for (int c = tid; c < cols; c += kThreads) {
                const unsigned long long kc = cand_key(zbuf[c], v0 + c);
                int rank = 0;
                for (int j = 0; j < cols; ++j) rank += cand_key(zbuf[j], v0 + j) > kc ? 1 : 0;
                if (rank < k) cand[atomicAdd(&n_cand, 1)] = kc;
            }
            if (tid == 0) expanded[t] = 1;
            __syncthreads();
        }
        n_expanded += nf;
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

size_t merge_smem_bytes(int n_tiles) {
    return static_cast<size_t>(n_tiles) * sizeof(Partial) +
           static_cast<size_t>(n_tiles * kListLen + kMergeExpandLists * kMaxK + n_tiles) * sizeof(unsigned long long) +
           static_cast<size_t>(n_tiles + 15) / 16 * 16;
}

cudaError_t launch_lmhead_merge(const Ctx& ctx, int dtype, const Partial* partials, int n_rows, int V, int d, int k,
                                float inv_temp, const void* lm_head, const void* x, int32_t* out_ids,
                                float* out_logp) {
    if (n_rows <= 0) return cudaSuccess;
    const int n_tiles = (V + kBlockV - 1) / kBlockV;
    const size_t smem = merge_smem_bytes(n_tiles);
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
