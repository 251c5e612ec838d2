// Merge of the LM-head partials into log-softmax top-k (Algorithm 1 "TopM" of stage 1 and the
// log-softmax + top-k of every stage-2 row).
//
// One CTA per row. The CTA
//   1. combines the row's half-block (max, sum of exp) pairs into its log-sum-exp and forms one
//      key (value desc, id asc) per half block from the half's best entry;
//   2. finds theta0, the k-th largest half-block key. Exactly the k halves at or above it can
//      hold members of the top k (every key elsewhere is below its half's best, hence below
//      theta0). Their chunks' two largest entries at or above theta0 are the candidates; the
//      k-th largest candidate key comes from a radix select over 64-bit keys;
//   3. certifies the result: a chunk whose third-largest value reaches the k-th candidate may
//      hide further members of the top k. Those chunks' 32 logits are recomputed exactly from
//      lm_head and x (in rounds of at most 64 chunks), replace the chunk's two candidates, and
//      the selection is redone;
//   4. writes the k winners sorted, as (id, logit - LSE).
// The result is the exact top-k of the full vocabulary whatever the input; a recompute needs
// three members of the top k in one 32-column chunk (about one row in 500 on random data).
#include <math.h>

#include "common.cuh"

namespace tf {
namespace {

constexpr int kThreads = 256;   // 512 or more: two CTAs no longer fit an SM, so 241 rows take two waves

__device__ __forceinline__ void lse_combine(float& m, float& s, float m2, float s2) {
    if (m2 > m) {
        s = s * __expf(m - m2) + s2;
        m = m2;
    } else if (m2 > -INFINITY) {
        s += s2 * __expf(m2 - m);
    }
}

// k-th largest of keys[0..n) (n >= k >= 1), by 8-bit digits from the most significant byte. Once
// the chosen digit's bin holds a single key, that key is the answer and is looked up directly
// (float keys of one row share their top bytes, so this usually ends the search after two or
// three digits instead of eight).
__device__ unsigned long long block_kth_largest(const unsigned long long* keys, int n, int k, int* hist,
                                                int* sel, unsigned long long* found) {
    unsigned long long prefix = 0;
    int rem = k;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    for (int shift = 56; shift >= 0; shift -= 8) {
        for (int i = tid; i < 256; i += kThreads) hist[i] = 0;
        __syncthreads();
        const unsigned long long hi_mask = shift == 56 ? 0ull : (~0ull << (shift + 8));
        // shared-memory atomics: lanes of a warp on one bin are combined by the hardware (a
        // warp match to aggregate them first costs far more on GB300)
        for (int i = tid; i < n; i += kThreads) {
            const unsigned long long key = keys[i];
            if ((key & hi_mask) == prefix) atomicAdd(&hist[static_cast<int>((key >> shift) & 255)], 1);
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
                        sel[0] = lane * 8 + b;
                        sel[1] = rem - c;
                        sel[2] = local[b];
                        break;
                    }
                    c += local[b];
                }
            }
        }
        __syncthreads();
        prefix |= static_cast<unsigned long long>(sel[0]) << shift;
        rem = sel[1];
        if (sel[2] == 1 && shift > 0) {
            // the k-th key is the only key with this prefix
            const unsigned long long mask = ~0ull << shift;
            for (int i = tid; i < n; i += kThreads)
                if ((keys[i] & mask) == prefix) *found = keys[i];
            __syncthreads();
            const unsigned long long r = *found;
            __syncthreads();   // every thread has read *found and sel before either is reused
            return r;
        }
        __syncthreads();       // every thread has read sel before the next digit rewrites it
    }
    return prefix;
}

// Shared state of block_kth_largest_fast.
constexpr int kBuckets = 256;
constexpr int kCollectCap = 256;
struct SelectSmem {
    int hist[kBuckets];
    unsigned long long coll[kCollectCap];
    float wmax[kThreads / 32], wmin[kThreads / 32];
    int wcnt[kThreads / 32];
    float vmin, scale;
    int total, bucket, rem, count, n_coll;
    unsigned long long found;
};

// The k-th largest non-zero key of keys[0..n) (zero keys are empty slots and rank below all),
// or 0 when fewer than k keys are non-zero. One histogram pass over 256 equal-width buckets of
// the key values (a monotone map, so the k-th largest key lies in the bucket where the count from
// the top reaches k), then an exact rank among the few keys of that bucket. Falls back to the
// byte-wise radix select when the values are all equal, not finite, or crowd one bucket.
__device__ unsigned long long block_kth_largest_fast(const unsigned long long* keys, int n, int k, SelectSmem& B,
                                                     int* hist, int* sel, unsigned long long* found) {
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    float vmax = -INFINITY, vmin = INFINITY;
    int cnt = 0;
    for (int i = tid; i < n; i += kThreads) {
        const unsigned long long key = keys[i];
        if (key != 0ull) {
            const float v = key_value(key);
            vmax = fmaxf(vmax, v);
            vmin = fminf(vmin, v);
            ++cnt;
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        vmax = fmaxf(vmax, __shfl_xor_sync(0xffffffffu, vmax, o));
        vmin = fminf(vmin, __shfl_xor_sync(0xffffffffu, vmin, o));
        cnt += __shfl_xor_sync(0xffffffffu, cnt, o);
    }
    if (lane == 0) {
        B.wmax[warp] = vmax;
        B.wmin[warp] = vmin;
        B.wcnt[warp] = cnt;
    }
    for (int i = tid; i < kBuckets; i += kThreads) B.hist[i] = 0;
    __syncthreads();
    if (warp == 0) {
        float mx = lane < kThreads / 32 ? B.wmax[lane] : -INFINITY;
        float mn = lane < kThreads / 32 ? B.wmin[lane] : INFINITY;
        int c = lane < kThreads / 32 ? B.wcnt[lane] : 0;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
            mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, o));
            c += __shfl_xor_sync(0xffffffffu, c, o);
        }
        if (lane == 0) {
            B.total = c;
            B.vmin = mn;
            const float range = mx - mn;
            B.scale = (range > 0.0f && isfinite(range)) ? static_cast<float>(kBuckets) / range : 0.0f;
            B.n_coll = 0;
        }
    }
    __syncthreads();
    const int total = B.total;
    const float scale = B.scale, vlo = B.vmin;
    if (total < k) {
        __syncthreads();
        return 0ull;
    }
    if (scale == 0.0f) {
        __syncthreads();
        return block_kth_largest(keys, n, k, hist, sel, found);
    }
    auto bucket_of = [&](unsigned long long key) {
        const int b = static_cast<int>((key_value(key) - vlo) * scale);
        return b < 0 ? 0 : (b >= kBuckets ? kBuckets - 1 : b);
    };
    for (int i = tid; i < n; i += kThreads) {
        const unsigned long long key = keys[i];
        if (key != 0ull) atomicAdd(&B.hist[bucket_of(key)], 1);
    }
    __syncthreads();
    if (warp == 0) {
        // lane l holds buckets 8l .. 8l+7; inclusive suffix sums over lanes (high buckets first)
        int local[8];
        int sum = 0;
#pragma unroll
        for (int b = 0; b < 8; ++b) {
            local[b] = B.hist[lane * 8 + b];
            sum += local[b];
        }
        int incl = sum;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int v = __shfl_down_sync(0xffffffffu, incl, o);
            if (lane + o < 32) incl += v;
        }
        const int excl = incl - sum;
        if (excl < k && k <= incl) {
            int c = excl;
            for (int b = 7; b >= 0; --b) {
                if (c + local[b] >= k) {
                    B.bucket = lane * 8 + b;
                    B.rem = k - c;
                    B.count = local[b];
                    break;
                }
                c += local[b];
            }
        }
    }
    __syncthreads();
    const int bk = B.bucket, rem = B.rem, cb = B.count;
    if (cb > kCollectCap) {
        __syncthreads();
        return block_kth_largest(keys, n, k, hist, sel, found);
    }
    for (int i = tid; i < n; i += kThreads) {
        const unsigned long long key = keys[i];
        if (key != 0ull && bucket_of(key) == bk) B.coll[atomicAdd(&B.n_coll, 1)] = key;
    }
    __syncthreads();
    // keys are distinct: exactly one has rem - 1 larger keys in the bucket
    for (int i = tid; i < cb; i += kThreads) {
        const unsigned long long key = B.coll[i];
        int rank = 0;
        for (int j = 0; j < cb; ++j) rank += B.coll[j] > key ? 1 : 0;
        if (rank == rem - 1) B.found = key;
    }
    __syncthreads();
    const unsigned long long r = B.found;
    __syncthreads();   // every thread has read the shared results before they are reused
    return r;
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

// Shared-memory layout of one merge CTA (dynamic part), for a top-k of k.
struct MergeSmem {
    unsigned long long* hkey;   // [n_halves] best key of every half block (0 = empty)
    unsigned long long* cand;   // [2 * 4k + kMergeExpandChunks * kChunk]
    unsigned long long* cand2;  // the same size: the compacted set of the next round
    unsigned long long* sel;    // [k] the winners
    float* c3;                  // [4k] third value of each kept chunk (bound on the rest)
    int* cbase;                 // [4k] first vocabulary id of each kept chunk
    int* chalf;                 // [k] the halves at or above theta0
    uint8_t* expanded;          // [4k] chunk recomputed
    float* xs;                  // [d] x of the row in fp32, staged only for a recompute
};
__host__ __device__ inline size_t merge_layout(int n_tiles, int d, int k, uint8_t* base, MergeSmem* m) {
    const size_t detail = static_cast<size_t>(k) * (kChunks / 2);   // chunks of the k halves kept
    size_t off = 0;
    auto take = [&](size_t bytes) {
        uint8_t* p = base ? base + off : nullptr;
        off += (bytes + 15) / 16 * 16;
        return p;
    };
    uint8_t* hk = take(static_cast<size_t>(2) * n_tiles * 8);
    uint8_t* cd = take((2 * detail + static_cast<size_t>(kMergeExpandChunks) * kChunk) * 8);
    uint8_t* cd2 = take((2 * detail + static_cast<size_t>(kMergeExpandChunks) * kChunk) * 8);
    uint8_t* se = take(static_cast<size_t>(k) * 8);
    uint8_t* c3 = take(detail * 4);
    uint8_t* cb = take(detail * 4);
    uint8_t* ch = take(static_cast<size_t>(k) * 4);
    uint8_t* ex = take(detail);
    uint8_t* xs = take(static_cast<size_t>(d) * 4);
    if (m) {
        m->hkey = reinterpret_cast<unsigned long long*>(hk);
        m->cand = reinterpret_cast<unsigned long long*>(cd);
        m->cand2 = reinterpret_cast<unsigned long long*>(cd2);
        m->sel = reinterpret_cast<unsigned long long*>(se);
        m->c3 = reinterpret_cast<float*>(c3);
        m->cbase = reinterpret_cast<int*>(cb);
        m->chalf = reinterpret_cast<int*>(ch);
        m->expanded = ex;
        m->xs = reinterpret_cast<float*>(xs);
    }
    return off;
}

template <typename T>
__global__ void __launch_bounds__(kThreads) lmhead_merge_kernel(Partials partials, int n_rows, int n_tiles, int V,
                                                                int d, int k, float inv_temp,
                                                                const T* __restrict__ lm_head,
                                                                const T* __restrict__ x, int32_t* __restrict__ out_ids,
                                                                float* __restrict__ out_logp, int* status) {
    pdl_trigger();
    pdl_wait();
    extern __shared__ __align__(16) uint8_t dsm[];
    MergeSmem S;
    merge_layout(n_tiles, d, k, dsm, &S);
    const int n_detail = k * (kChunks / 2);
    __shared__ int hist[256];
    __shared__ SelectSmem SB;
    __shared__ float red_m[kThreads / 32], red_s[kThreads / 32];
    __shared__ int sel_info[3], n_flag, flag_list[kMergeExpandChunks], n_cand, n_next, n_sel, n_valid, n_chalf;
    __shared__ unsigned long long found;
    __shared__ float zbuf[kMergeExpandChunks * kChunk];
    __shared__ float lse_s;

    const int row = blockIdx.x;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int nh = 2 * n_tiles;
    if (tid == 0) {
        n_cand = 0;
        n_valid = 0;
        n_chalf = 0;
    }

    // 1. half-block summaries (strided by n_rows, eight loads in flight per thread): the row's
    //    log-sum-exp and one key per half
    float m = -INFINITY, s = 0.0f;
    int my_valid = 0;
    {
        const float4* src = partials.halves + row;
        const size_t stride = static_cast<size_t>(partials.n_rows);
        for (int base = tid; base < nh; base += 8 * kThreads) {
            float4 v[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int i = base + j * kThreads;
                if (i < nh) v[j] = src[static_cast<size_t>(i) * stride];
            }
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int i = base + j * kThreads;
                if (i >= nh) break;
                const int id = __float_as_int(v[j].w);
                unsigned long long key = 0ull;
                if (id >= 0) {
                    lse_combine(m, s, v[j].x, v[j].y);
                    key = cand_key(v[j].z, id);
                    ++my_valid;
                }
                S.hkey[i] = key;
            }
        }
    }
    for (int i = tid; i < n_detail; i += kThreads) S.expanded[i] = 0;
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
    __syncthreads();
    atomicAdd(&n_valid, my_valid);
    __syncthreads();
    if (warp == 0) {
        float M = lane < kThreads / 32 ? red_m[lane] : -INFINITY;
        float Ssum = lane < kThreads / 32 ? red_s[lane] : 0.0f;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float m2 = __shfl_xor_sync(0xffffffffu, M, o);
            const float s2 = __shfl_xor_sync(0xffffffffu, Ssum, o);
            lse_combine(M, Ssum, m2, s2);
        }
        if (lane == 0) {
            const float lse = M + logf(Ssum);
            lse_s = lse;
            if (!isfinite(lse)) set_status(status, TF_DEV_NONFINITE);
        }
    }

    // 2. theta0 and the halves at or above it (at most k: the keys are distinct)
    const unsigned long long theta0 =
        n_valid >= k ? block_kth_largest_fast(S.hkey, nh, k, SB, hist, sel_info, &found) : 0ull;
    for (int i = tid; i < nh; i += kThreads) {
        const unsigned long long key = S.hkey[i];
        if (key != 0ull && key >= theta0) {
            const int slot = atomicAdd(&n_chalf, 1);
            if (slot < k) S.chalf[slot] = i;
        }
    }
    __syncthreads();
    const int nch = min(n_chalf, k);
    // their chunks: the two largest entries at or above theta0 become candidates
    for (int i = tid; i < nch * (kChunks / 2); i += kThreads) {
        const int h = S.chalf[i >> 2];
        const int tile = h >> 1, chunk = (h & 1) * (kChunks / 2) + (i & 3);
        const float4 q = partials.chunks[partials.chunk_at(tile, chunk, row)];
        const int v0 = tile * kBlockV + chunk * kChunk;
        const int ids = __float_as_int(q.w);
        S.cbase[i] = v0;
        S.c3[i] = q.z;
        if (q.x > -INFINITY) {
            const unsigned long long key = cand_key(q.x, v0 + (ids & 255));
            if (key >= theta0) S.cand[atomicAdd(&n_cand, 1)] = key;
        }
        if (q.y > -INFINITY) {
            const unsigned long long key = cand_key(q.y, v0 + ((ids >> 8) & 255));
            if (key >= theta0) S.cand[atomicAdd(&n_cand, 1)] = key;
        }
    }
    __syncthreads();

    // 3. select; a kept chunk whose third value reaches the k-th candidate may hide members of
    //    the top k, so its 32 logits are recomputed exactly and the selection is redone. Chunks
    //    are recomputed in rounds of at most kMergeExpandChunks; after each round only keys at or
    //    above the k-th candidate survive (the candidates are logits of the row, so every member
    //    of the true top k is at or above it, and it only rises), which bounds the set by
    //    k + kMergeExpandChunks * kChunk whatever the input.
    bool x_staged = false;
    unsigned long long theta = 0;
    unsigned long long* cand = S.cand;
    unsigned long long* spare = S.cand2;
    for (;;) {
        const int nc = n_cand;
        theta = nc >= k ? block_kth_largest_fast(cand, nc, k, SB, hist, sel_info, &found) : 0ull;
        const float tval = key_value(theta);
        if (tid == 0) n_flag = 0;
        __syncthreads();
        for (int i = tid; i < nch * (kChunks / 2); i += kThreads) {
            if (S.expanded[i] || !(S.c3[i] > -INFINITY)) continue;
            if (nc < k || S.c3[i] >= tval) {
                const int slot = atomicAdd(&n_flag, 1);
                if (slot < kMergeExpandChunks) flag_list[slot] = i;
            }
        }
        __syncthreads();
        const int nf = min(n_flag, kMergeExpandChunks);   // the rest wait for the next round
        if (nf == 0) break;
        if (tid == 0) {
            set_status(status, TF_DEV_RECOMPUTED);
            n_next = 0;
        }
        // exact logits of this round's chunks: x staged once in shared memory, then one warp per
        // column with all of its 16-byte weight loads issued before the multiply-adds
        if (!x_staged) {
            for (int i = tid; i < d; i += kThreads) S.xs[i] = to_f32(x[static_cast<size_t>(row) * d + i]);
            x_staged = true;
        }
        __syncthreads();
        for (int q = warp; q < nf * kChunk; q += kThreads / 32) {
            const int f = q / kChunk, cc = q - f * kChunk;
            const int v = S.cbase[flag_list[f]] + cc;
            const float acc = v < V ? dot_row(lm_head + static_cast<size_t>(v) * d, S.xs, d, lane) : 0.0f;
            if (lane == 0) zbuf[q] = v < V ? acc * inv_temp : -INFINITY;
        }
        __syncthreads();
        // the next set: surviving keys not from this round's chunks, then their exact logits
        for (int j = tid; j < nc; j += kThreads) {
            const unsigned long long key = cand[j];
            if (key == 0ull || key < theta) continue;
            const int id = key_id(key);
            bool mine = false;
            for (int f = 0; f < nf; ++f) {
                const int v0 = S.cbase[flag_list[f]];
                mine = mine || (id >= v0 && id < v0 + kChunk);
            }
            if (!mine) spare[atomicAdd(&n_next, 1)] = key;
        }
        for (int q = tid; q < nf * kChunk; q += kThreads) {
            const int f = q / kChunk, cc = q - f * kChunk;
            const int v = S.cbase[flag_list[f]] + cc;
            if (v < V) {
                const unsigned long long key = cand_key(zbuf[q], v);
                if (key >= theta) spare[atomicAdd(&n_next, 1)] = key;
            }
        }
        for (int f = tid; f < nf; f += kThreads) S.expanded[flag_list[f]] = 1;
        __syncthreads();
        if (tid == 0) n_cand = n_next;
        unsigned long long* t = cand;
        cand = spare;
        spare = t;
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
            if (slot < k) S.sel[slot] = key;
        }
    }
    __syncthreads();
    const int ns = min(n_sel, k);
    const float lse = lse_s;
    for (int i = tid; i < ns; i += kThreads) {
        const unsigned long long key = S.sel[i];
        int rank = 0;
        for (int j = 0; j < ns; ++j) rank += S.sel[j] > key ? 1 : 0;
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

size_t merge_smem_bytes(int n_tiles, int d, int k) { return merge_layout(n_tiles, d, k, nullptr, nullptr); }

cudaError_t launch_lmhead_merge(const Ctx& ctx, int dtype, Partials partials, int n_rows, int V, int d, int k,
                                float inv_temp, const void* lm_head, const void* x, int32_t* out_ids,
                                float* out_logp) {
    if (n_rows <= 0) return cudaSuccess;
    const int n_tiles = (V + kBlockV - 1) / kBlockV;
    const size_t smem = merge_smem_bytes(n_tiles, d, k);
    if (dtype == TF_BF16) {
        auto kern = lmhead_merge_kernel<__nv_bfloat16>;
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
        if (e != cudaSuccess) return e;
        e = launch_pdl(kern, dim3(n_rows), dim3(kThreads), smem, ctx.stream, partials, n_rows, n_tiles, V, d, k,
                       inv_temp, static_cast<const __nv_bfloat16*>(lm_head), static_cast<const __nv_bfloat16*>(x),
                       out_ids, out_logp, ctx.status);
        if (e != cudaSuccess) return e;
    } else {
        auto kern = lmhead_merge_kernel<float>;
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
        if (e != cudaSuccess) return e;
        e = launch_pdl(kern, dim3(n_rows), dim3(kThreads), smem, ctx.stream, partials, n_rows, n_tiles, V, d, k,
                       inv_temp, static_cast<const float*>(lm_head), static_cast<const float*>(x), out_ids, out_logp,
                       ctx.status);
        if (e != cudaSuccess) return e;
    }
    return cudaGetLastError();
}

}  // namespace tf
