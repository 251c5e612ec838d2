// Stage-2 input rows (Eq. 1), Part 2 of Algorithm 1 (OPT-Tree best-first selection) and the
// verifier's tree-attention mask.
#include <math.h>

#include "common.cuh"

namespace tf {
namespace {

// ------------------------------------------------------------------------------------------
// x = [RMSNorm(h_{t+i}) * norm_h ; RMSNorm(Embd(prev)) * norm_e] for every stage-2 row
// (Eq. 1, h~ first). One CTA per row; the embedding row is gathered by token id here, so
// the candidate embeddings are never materialised on their own.
// ------------------------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(256) gather_norm_kernel(const T* __restrict__ hidden, const T* __restrict__ embed,
                                                          const T* __restrict__ norm_h, const T* __restrict__ norm_e,
                                                          const int32_t* __restrict__ root_tok,
                                                          const int32_t* __restrict__ top_ids, int gamma, int M,
                                                          int K1, int R, int d, int V, float eps, T* __restrict__ X,
                                                          int* status) {
    __shared__ float red[2][8];
    const int row = blockIdx.x;
    const int sq = row / R, r = row - sq * R;
    const int hid = sq * gamma + stage2_hidden_index(r, M);
    int tok = (r == 0) ? root_tok[sq] : top_ids[(static_cast<size_t>(sq) * gamma + (r - 1) / M) * K1 + (r - 1) % M];
    if (tok < 0 || tok >= V) {
        if (threadIdx.x == 0) set_status(status, TF_DEV_BAD_TOKEN);
        tok = 0;
    }
    const T* h = hidden + static_cast<size_t>(hid) * d;
    const T* e = embed + static_cast<size_t>(tok) * d;
    float sh = 0.0f, se = 0.0f;
    for (int k = threadIdx.x; k < d; k += blockDim.x) {
        const float a = to_f32(h[k]), b = to_f32(e[k]);
        sh = fmaf(a, a, sh);
        se = fmaf(b, b, se);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        sh += __shfl_xor_sync(0xffffffffu, sh, o);
        se += __shfl_xor_sync(0xffffffffu, se, o);
    }
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) {
        red[0][warp] = sh;
        red[1][warp] = se;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        float a = 0.0f, b = 0.0f;
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w) {
            a += red[0][w];
            b += red[1][w];
        }
        red[0][0] = rsqrtf(a / d + eps);
        red[1][0] = rsqrtf(b / d + eps);
    }
    __syncthreads();
    const float ih = red[0][0], ie = red[1][0];
    T* xr = X + static_cast<size_t>(row) * 2 * d;
    for (int k = threadIdx.x; k < d; k += blockDim.x) {
        xr[k] = from_f32<T>(to_f32(h[k]) * ih * to_f32(norm_h[k]));
        xr[d + k] = from_f32<T>(to_f32(e[k]) * ie * to_f32(norm_e[k]));
    }
}

// ------------------------------------------------------------------------------------------
// OPT-Tree selection, one warp per sequence. The queue holds one entry per open child list:
// (score, parent score, parent node, list row, rank in the list, depth, token). Popping rank k
// of a list replaces the entry by rank k+1 of the same list (its next sibling), and an
// expandable popped node adds rank 0 of its own child list. Because every list is sorted
// (value desc, id asc), this pops exactly what pushing whole distributions would (Algorithm 1
// Part 2 pushes q'^(m) entirely), with at most B + 1 entries live at any time.
// ------------------------------------------------------------------------------------------
struct TreeArgs {
    int gamma, M, K1, K2, B, V, mode, R;
    const int32_t* root_tok;
    const int32_t* top_ids;
    const float* top_logp;
    const int32_t* child_ids;
    const float* child_logp;
    int32_t* node_tok;
    int32_t* node_parent;
    int32_t* node_depth;
    float* node_score;
    int32_t* dev_status;
};

struct Q {
    float* score;
    float* pscore;
    int* parent;
    int* row;
    int* rank;
    int* depth;
    int* tok;
};

__device__ __forceinline__ bool q_better(const Q& q, int a, int b) {
    if (b < 0) return a >= 0;
    if (a < 0) return false;
    if (q.score[a] != q.score[b]) return q.score[a] > q.score[b];
    if (q.depth[a] != q.depth[b]) return q.depth[a] < q.depth[b];
    if (q.parent[a] != q.parent[b]) return q.parent[a] < q.parent[b];
    return q.tok[a] < q.tok[b];
}

__global__ void __launch_bounds__(32) build_tree_kernel(TreeArgs a) {
    extern __shared__ uint8_t smem_raw[];
    const int cap = a.B + 2;
    Q q;
    q.score = reinterpret_cast<float*>(smem_raw);
    q.pscore = q.score + cap;
    q.parent = reinterpret_cast<int*>(q.pscore + cap);
    q.row = q.parent + cap;
    q.rank = q.row + cap;
    q.depth = q.rank + cap;
    q.tok = q.depth + cap;

    const int s = blockIdx.x;
    const int lane = threadIdx.x;
    const int n_out = a.B + 1;
    int flags = 0;
    const int root = a.root_tok[s];
    if (root < 0 || root >= a.V) flags |= TF_DEV_BAD_TOKEN;

    const bool ar = a.mode == TF_MODE_AR;
    const int list_len = a.K2;
    // child list `row` of this sequence: stage-2 rows (AR) or stage-1 depths (marginal modes)
    auto ids_of = [&](int row) -> const int32_t* {
        return ar ? a.child_ids + (static_cast<size_t>(s) * a.R + row) * a.K2
                  : a.top_ids + (static_cast<size_t>(s) * a.gamma + row) * a.K1;
    };
    auto lp_of = [&](int row) -> const float* {
        return ar ? a.child_logp + (static_cast<size_t>(s) * a.R + row) * a.K2
                  : a.top_logp + (static_cast<size_t>(s) * a.gamma + row) * a.K1;
    };

    int n_e = 0;
    if (lane == 0) {
        a.node_tok[static_cast<size_t>(s) * n_out] = root;
        a.node_parent[static_cast<size_t>(s) * n_out] = -1;
        a.node_depth[static_cast<size_t>(s) * n_out] = 0;
        a.node_score[static_cast<size_t>(s) * n_out] = 0.0f;
        const float lp = lp_of(0)[0];
        q.score[0] = lp;
        q.pscore[0] = 0.0f;
        q.parent[0] = 0;
        q.row[0] = 0;
        q.rank[0] = 0;
        q.depth[0] = 1;
        q.tok[0] = ids_of(0)[0];
    }
    n_e = 1;
    __syncwarp();

    int count = 1;
    while (count < n_out && n_e > 0) {
        // warp-wide arg-max over live entries in the queue order
        int best = -1;
        for (int j = lane; j < n_e; j += 32)
            if (q_better(q, j, best)) best = j;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const int other = __shfl_xor_sync(0xffffffffu, best, o);
            if (q_better(q, other, best)) best = other;
        }
        const float sc = q.score[best], psc = q.pscore[best];
        const int par = q.parent[best], row = q.row[best], rank = q.rank[best];
        const int dep = q.depth[best], tok = q.tok[best];
        __syncwarp();
        const int node = count++;
        if (tok < 0 || tok >= a.V) flags |= TF_DEV_BAD_TOKEN;
        if (!isfinite(sc)) flags |= TF_DEV_NONFINITE;
        // expandable? (depth cap; M-ary rule via one compare per lane)
        int crow = -1;
        if (dep < a.gamma) {
            if (a.mode == TF_MODE_MARGINAL) {
                crow = dep;
            } else {
                const bool hit = lane < a.M &&
                                 a.top_ids[(static_cast<size_t>(s) * a.gamma + dep - 1) * a.K1 + lane] == tok;
                const unsigned bal = __ballot_sync(0xffffffffu, hit);
                if (bal) {
                    const int m = __ffs(bal) - 1;
                    crow = ar ? 1 + (dep - 1) * a.M + m : dep;
                }
            }
        }
        if (lane == 0) {
            const size_t o = static_cast<size_t>(s) * n_out + node;
            a.node_tok[o] = tok;
            a.node_parent[o] = par;
            a.node_depth[o] = dep;
            a.node_score[o] = sc;
            if (rank + 1 < list_len) {       // next sibling of the popped entry
                q.rank[best] = rank + 1;
                q.tok[best] = ids_of(row)[rank + 1];
                q.score[best] = psc + lp_of(row)[rank + 1];
            } else {                         // list exhausted: move the last entry here
                const int last = n_e - 1;
                q.score[best] = q.score[last];
                q.pscore[best] = q.pscore[last];
                q.parent[best] = q.parent[last];
                q.row[best] = q.row[last];
                q.rank[best] = q.rank[last];
                q.depth[best] = q.depth[last];
                q.tok[best] = q.tok[last];
            }
        }
        if (rank + 1 >= list_len) --n_e;
        if (crow >= 0) {
            if (lane == 0) {
                q.score[n_e] = sc + lp_of(crow)[0];
                q.pscore[n_e] = sc;
                q.parent[n_e] = node;
                q.row[n_e] = crow;
                q.rank[n_e] = 0;
                q.depth[n_e] = dep + 1;
                q.tok[n_e] = ids_of(crow)[0];
            }
            ++n_e;
        }
        __syncwarp();
    }
    if (count < n_out) flags |= TF_DEV_UNDERFULL;
    for (int i = count + lane; i < n_out; i += 32) {
        const size_t o = static_cast<size_t>(s) * n_out + i;
        a.node_tok[o] = -1;
        a.node_parent[o] = -1;
        a.node_depth[o] = -1;
        a.node_score[o] = -INFINITY;
    }
    if (lane == 0) a.dev_status[s] = flags;
}

// ------------------------------------------------------------------------------------------
// mask[i][j] = 1 iff node j is node i or one of its ancestors. Ancestor sets are bitsets built
// level by level (a node's set is its parent's set plus itself); pos = root_pos + depth.
// Nodes with an invalid parent link (missing nodes) get empty rows and columns and pos -1.
// ------------------------------------------------------------------------------------------
__global__ void __launch_bounds__(256) tree_mask_kernel(int n, const int32_t* __restrict__ node_parent,
                                                        const int32_t* __restrict__ node_depth,
                                                        const int32_t* __restrict__ root_pos,
                                                        uint8_t* __restrict__ mask, int32_t* __restrict__ pos_ids) {
    extern __shared__ uint32_t sm[];
    const int W = (n + 31) / 32;
    int* par = reinterpret_cast<int*>(sm);
    int* dep = par + n;
    uint32_t* anc = reinterpret_cast<uint32_t*>(dep + n);
    __shared__ int max_dep;
    const int s = blockIdx.x;
    const int32_t* P = node_parent + static_cast<size_t>(s) * n;
    const int32_t* D = node_depth + static_cast<size_t>(s) * n;
    if (threadIdx.x == 0) max_dep = 0;
    for (int i = threadIdx.x; i < n * W; i += blockDim.x) anc[i] = 0u;
    __syncthreads();
    for (int i = threadIdx.x; i < n; i += blockDim.x) {
        int p = P[i], d = D[i];
        const bool ok = (i == 0) ? (d == 0) : (p >= 0 && p < i && d >= 1 && d <= kMaxGamma);
        par[i] = ok ? p : -1;
        dep[i] = ok ? d : -1;
        if (ok) atomicMax(&max_dep, d);
    }
    __syncthreads();
    for (int L = 0; L <= max_dep; ++L) {
        for (int idx = threadIdx.x; idx < n * W; idx += blockDim.x) {
            const int i = idx / W, w = idx - (idx / W) * W;
            if (dep[i] != L) continue;
            uint32_t v = 0u;
            if (L > 0) {
                const int p = par[i];
                // the parent must sit one level up and be present (its own bit set)
                if (dep[p] != L - 1 || !((anc[p * W + p / 32] >> (p & 31)) & 1u)) continue;
                v = anc[p * W + w];
            }
            if (w == i / 32) v |= 1u << (i & 31);
            anc[i * W + w] = v;
        }
        __syncthreads();
    }
    uint8_t* out = mask + static_cast<size_t>(s) * n * n;
    for (int idx = threadIdx.x; idx < n * n; idx += blockDim.x) {
        const int i = idx / n, j = idx - (idx / n) * n;
        out[idx] = static_cast<uint8_t>((anc[i * W + j / 32] >> (j & 31)) & 1u);
    }
    for (int i = threadIdx.x; i < n; i += blockDim.x) {
        const bool present = (anc[i * W + i / 32] >> (i & 31)) & 1u;
        pos_ids[static_cast<size_t>(s) * n + i] = present ? root_pos[s] + dep[i] : -1;
    }
}

}  // namespace

cudaError_t launch_gather_norm(const Ctx& ctx, int dtype, const void* hidden, const void* embed, const void* norm_h,
                               const void* norm_e, const int32_t* root_tok, const int32_t* top_ids, int b, int gamma,
                               int M, int K1, int d, int V, float eps, void* X) {
    const int R = 1 + M * (gamma - 1);
    const int rows = b * R;
    if (dtype == TF_BF16) {
        gather_norm_kernel<__nv_bfloat16><<<rows, 256, 0, ctx.stream>>>(
            static_cast<const __nv_bfloat16*>(hidden), static_cast<const __nv_bfloat16*>(embed),
            static_cast<const __nv_bfloat16*>(norm_h), static_cast<const __nv_bfloat16*>(norm_e), root_tok, top_ids,
            gamma, M, K1, R, d, V, eps, static_cast<__nv_bfloat16*>(X), ctx.status);
    } else {
        gather_norm_kernel<float><<<rows, 256, 0, ctx.stream>>>(
            static_cast<const float*>(hidden), static_cast<const float*>(embed), static_cast<const float*>(norm_h),
            static_cast<const float*>(norm_e), root_tok, top_ids, gamma, M, K1, R, d, V, eps,
            static_cast<float*>(X), ctx.status);
    }
    return cudaGetLastError();
}

cudaError_t launch_build_tree(const Ctx& ctx, int b, int gamma, int M, int K1, int K2, int B, int V, int mode, int R,
                              const int32_t* root_tok, const int32_t* top_ids, const float* top_logp,
                              const int32_t* child_ids, const float* child_logp, int32_t* node_tok,
                              int32_t* node_parent, int32_t* node_depth, float* node_score, int32_t* dev_status) {
    TreeArgs a{gamma, M, K1, K2, B, V, mode, R, root_tok, top_ids, top_logp, child_ids, child_logp,
               node_tok, node_parent, node_depth, node_score, dev_status};
    const size_t smem = static_cast<size_t>(B + 2) * 7 * 4;
    cudaError_t e = cudaFuncSetAttribute(build_tree_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    build_tree_kernel<<<b, 32, smem, ctx.stream>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_tree_mask(const Ctx& ctx, int b, int B, const int32_t* node_parent, const int32_t* node_depth,
                             const int32_t* root_pos, uint8_t* mask, int32_t* pos_ids) {
    const int n = B + 1;
    const int W = (n + 31) / 32;
    const size_t smem = static_cast<size_t>(2 * n + n * W) * 4;
    cudaError_t e = cudaFuncSetAttribute(tree_mask_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    tree_mask_kernel<<<b, 256, smem, ctx.stream>>>(n, node_parent, node_depth, root_pos, mask, pos_ids);
    return cudaGetLastError();
}

}  // namespace tf
