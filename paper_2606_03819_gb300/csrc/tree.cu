// Stage-2 input rows (Eq. 1), Part 2 of Algorithm 1 (OPT-Tree best-first selection) and the
// verifier's tree-attention mask.
#include <math.h>

#include "common.cuh"

namespace tf {
namespace {

// ------------------------------------------------------------------------------------------
// Inputs of stage-2 row `row` (R rows per sequence).
//  TreeFlash (Eq. 1): row 0 refines depth 1 with the root token; row 1 + (i-2) M + m refines
//  depth i with candidate m of depth i-1.
//  Two previous tokens (the ablations' two-token variant): row 0 refines depth 1 with (x_t,
//  x_{t-1}) = root_tok[2 sq], root_tok[2 sq + 1]; rows 1..M depth 2 with (candidate m of depth 1,
//  x_t); row 1 + M + (i-3) M^2 + m1 M + m2 depth i >= 3 with (candidate m1 of depth i-1,
//  candidate m2 of depth i-2).
// The hidden-state index needs no kernel's output, so it is separate from the token reads.
// ------------------------------------------------------------------------------------------
__device__ __forceinline__ int stage2_row_hidden(int row, int R, int gamma, int M, bool two_prev) {
    const int sq = row / R, r = row - sq * R;
    if (!two_prev) return sq * gamma + stage2_hidden_index(r, M);
    const int depth = r == 0 ? 1 : r <= M ? 2 : 3 + (r - 1 - M) / (M * M);
    return sq * gamma + depth - 1;
}
// The previous token (p[0]) and, with two_prev, the one before it (p[1]).
__device__ __forceinline__ void stage2_row_tokens(int row, int R, int gamma, int M, int K1, bool two_prev,
                                                  const int32_t* root_tok, const int32_t* top_ids, int* p) {
    const int sq = row / R, r = row - sq * R;
    const int32_t* top = top_ids + static_cast<size_t>(sq) * gamma * K1;   // [gamma][K1] of this sequence
    if (!two_prev) {
        p[0] = r == 0 ? root_tok[sq] : top[((r - 1) / M) * K1 + (r - 1) % M];
        return;
    }
    const int32_t* root = root_tok + 2 * static_cast<size_t>(sq);
    if (r == 0) {
        p[0] = root[0];
        p[1] = root[1];
    } else if (r <= M) {
        p[0] = top[r - 1];
        p[1] = root[0];
    } else {
        const int q = r - 1 - M, i = 3 + q / (M * M), w = q - (i - 3) * M * M;
        p[0] = top[(i - 2) * K1 + w / M];
        p[1] = top[(i - 3) * K1 + w % M];
    }
}

// ------------------------------------------------------------------------------------------
// x = [RMSNorm(h_{t+i}) * norm_h ; RMSNorm(Embd(prev)) * norm_e] for every stage-2 row
// (Eq. 1, h~ first), and with NE = 2 a third part RMSNorm(Embd(token before prev)) * norm_e.
// One CTA per row; the embedding rows are gathered by token id here, so the candidate
// embeddings are never materialised on their own. hres (NE = 2): the row's hidden state.
// ------------------------------------------------------------------------------------------
template <typename T, int NE>
__global__ void __launch_bounds__(256) gather_norm_kernel(const T* __restrict__ hidden, const T* __restrict__ embed,
                                                          const T* __restrict__ norm_h, const T* __restrict__ norm_e,
                                                          const int32_t* __restrict__ root_tok,
                                                          const int32_t* __restrict__ top_ids, int gamma, int M,
                                                          int K1, int R, int d, int V, float eps, T* __restrict__ X,
                                                          T* __restrict__ hres, int* status) {
    pdl_trigger();
    pdl_wait();
    // the approximator GEMMs' tail-split counters (after the status word) start each call at zero
    if (blockIdx.x == 0 && status)
        for (int i = threadIdx.x; i < kTailSems; i += blockDim.x) status[1 + i] = 0;
    __shared__ float red[1 + NE][8];
    const int row = blockIdx.x;
    const int hid = stage2_row_hidden(row, R, gamma, M, NE == 2);
    int tok[2] = {0, 0};
    stage2_row_tokens(row, R, gamma, M, K1, NE == 2, root_tok, top_ids, tok);
    const T* seg[1 + NE];
    seg[0] = hidden + static_cast<size_t>(hid) * d;
#pragma unroll
    for (int j = 0; j < NE; ++j) {
        if (tok[j] < 0 || tok[j] >= V) {
            if (threadIdx.x == 0) set_status(status, TF_DEV_BAD_TOKEN);
            tok[j] = 0;
        }
        seg[1 + j] = embed + static_cast<size_t>(tok[j]) * d;
    }
    float sumsq[1 + NE];
#pragma unroll
    for (int j = 0; j <= NE; ++j) sumsq[j] = 0.0f;
    for (int k = threadIdx.x; k < d; k += blockDim.x) {
#pragma unroll
        for (int j = 0; j <= NE; ++j) {
            const float a = to_f32(seg[j][k]);
            sumsq[j] = fmaf(a, a, sumsq[j]);
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
#pragma unroll
        for (int j = 0; j <= NE; ++j) sumsq[j] += __shfl_xor_sync(0xffffffffu, sumsq[j], o);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0)
#pragma unroll
        for (int j = 0; j <= NE; ++j) red[j][warp] = sumsq[j];
    __syncthreads();
    if (threadIdx.x <= NE) {
        float a = 0.0f;
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w) a += red[threadIdx.x][w];
        red[threadIdx.x][0] = rsqrtf(a / d + eps);
    }
    __syncthreads();
    T* xr = X + static_cast<size_t>(row) * (1 + NE) * d;
    for (int k = threadIdx.x; k < d; k += blockDim.x) {
        const float hk = to_f32(seg[0][k]);
        xr[k] = from_f32<T>(hk * red[0][0] * to_f32(norm_h[k]));
#pragma unroll
        for (int j = 1; j <= NE; ++j) xr[j * d + k] = from_f32<T>(to_f32(seg[j][k]) * red[j][0] * to_f32(norm_e[k]));
        if (NE == 2) hres[static_cast<size_t>(row) * d + k] = seg[0][k];
    }
}

// ------------------------------------------------------------------------------------------
// OPT-Tree selection (Algorithm 1 Part 2), one warp per sequence. The queue holds one entry per
// open child list: (path score, depth, parent node) packed into one 64-bit key, plus the list
// row, the rank in the list, the parent's score and the token. Popping rank k of a list
// replaces the entry by rank k+1 of the same list (its next sibling), and an expandable popped
// node adds rank 0 of its own child list. Every list is sorted (value desc, id asc), so this
// pops exactly what pushing whole distributions would, with at most B + 1 live entries.
//
// Queue order: larger score, then smaller depth, then smaller parent index. Two live entries
// never share (depth, parent): each node opens at most one child list. So the key
//   float_key(score) << 32 | (127 - depth) << 24 | (0xFFFFFF - parent)
// is unique and its integer maximum is the next pop. Each lane keeps the best key of its own
// slots (j = lane mod 32) and rescans only when one of them changed; a pop is two warp max
// reductions and a ballot.
// ------------------------------------------------------------------------------------------
struct TreeArgs {
    int gamma, M, K1, K2, B, V, mode, R;
    int two_prev;      // child lists by the ablations' two-token rule; root_tok holds 2 tokens per sequence
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
    // optional, with B + 1 <= kMaskRows: the builder also writes the verification mask and
    // position ids (tf_tree_mask's outputs) from the tree it holds in shared memory
    const int32_t* root_pos;
    uint8_t* mask;
    int32_t* pos_ids;
    // optional: the workspace status word, final once the builder runs (every earlier kernel of
    // the step has finished). Each dev_status[s] then becomes seq_bits | w | w << 16 with w that
    // word, so that a caller that reads dev_status alone also learns w by itself.
    const int32_t* ws_status;
};

// The status word of sequence s: its own bits, and with a.ws_status the folded workspace word.
__device__ __forceinline__ int32_t sequence_status(const TreeArgs& a, int flags) {
    if (!a.ws_status) return flags;
    const int32_t w = *a.ws_status;
    return flags | w | (w << 16);
}

// Index m of `tok` among the M <= 64 stage-1 candidates of depth `dep` (the M-ary rule of
// Algorithm 1 Part 2: the node is expandable iff its token is one of them), or -1; two warp
// ballots, so every lane of the warp must call it (active = false gives -1).
__device__ __forceinline__ int mary_index(const int* topm, int dep, int M, int tok, int lane, bool active) {
    const int* t = topm + (dep - 1) * M;
    const bool h0 = active && lane < M && t[lane] == tok;
    const bool h1 = active && lane + 32 < M && t[lane + 32] == tok;
    const unsigned b0 = __ballot_sync(0xffffffffu, h0), b1 = __ballot_sync(0xffffffffu, h1);
    return b0 ? __ffs(b0) - 1 : (b1 ? 32 + __ffs(b1) - 1 : -1);
}

// Child list of a popped node under the two-previous-token rule: the node (depth dep, candidate
// m of its depth, or m < 0 outside the M-ary tree) gets the row conditioned on its own token and
// its parent's, 1 + m for dep = 1 and 1 + M + (dep - 2) M^2 + m M + mp for dep >= 2, mp the
// parent's candidate index at depth dep - 1 (the parent was expanded, so it has one). o_tok holds
// the tokens of the nodes placed so far, written by lane 0, which alone reads the parent's token.
// Every lane must call it (ballots); returns -1 for a leaf.
__device__ __forceinline__ int child_row_2prev(const int* topm, const int* o_tok, int M, int dep, int m, int par,
                                               int lane) {
    const bool deep = m >= 0 && dep >= 2;
    int ptok = 0;
    if (lane == 0 && deep) ptok = o_tok[par];
    ptok = __shfl_sync(0xffffffffu, ptok, 0);
    const int mp = mary_index(topm, deep ? dep - 1 : 1, M, ptok, lane, deep);
    if (m < 0) return -1;
    if (dep == 1) return 1 + m;
    return mp >= 0 ? 1 + M + (dep - 2) * M * M + m * M + mp : -1;
}

__device__ __forceinline__ unsigned long long queue_key(float score, int depth, int parent) {
    return (static_cast<unsigned long long>(float_key(score)) << 32) |
           (static_cast<unsigned long long>(127 - depth) << 24) | static_cast<unsigned long long>(0xFFFFFF - parent);
}

constexpr int kTreeThreads = 256;
constexpr int kMaskRows = kFusedMaskMaxNodes;    // mask rows per CTA (the fused mask is one block)

// Shared-memory bytes of build_tree_kernel: queue, node arrays, stage-1 top-M, and (when they
// fit) the sequence's child lists.
__host__ __device__ inline size_t tree_mask_words(int n) { return static_cast<size_t>(n) * ((n + 31) / 32); }
__host__ __device__ inline size_t tree_smem_fixed(int B, int gamma, int M, bool with_mask) {
    return static_cast<size_t>(B + 2) * (8 + 4 * 4) + static_cast<size_t>(B + 1) * 4 * 4 +
           static_cast<size_t>(gamma) * M * 4 + 16 + (with_mask ? tree_mask_words(B + 1) * 4 + 16 : 0);
}
// Bytes of the staged list prefixes: the first sw entries of each of the rows child lists.
__host__ __device__ inline size_t tree_smem_lists(int rows, int sw) { return static_cast<size_t>(rows) * sw * 8; }
constexpr size_t kTreeSmemLimit = 200 * 1024;

// The child lists of one sequence: the first sw entries of every row staged in shared memory,
// the rest read from global memory. A list's entry of rank r is reached only after r pops of
// that list, so sw = min(list length, B + 1) already covers every entry a tree can use.
struct ListView {
    const int32_t* s_ids;   // [rows][sw]
    const float* s_lp;
    const int32_t* g_ids;   // [rows][stride]
    const float* g_lp;
    int sw, stride;
    __device__ __forceinline__ int tok(int row, int rank) const {
        return rank < sw ? s_ids[row * sw + rank] : g_ids[static_cast<size_t>(row) * stride + rank];
    }
    __device__ __forceinline__ float lp(int row, int rank) const {
        return rank < sw ? s_lp[row * sw + rank] : g_lp[static_cast<size_t>(row) * stride + rank];
    }
};

// Shared memory of both builders: queue arrays (used by the general builder only), output nodes,
// stage-1 top-M and the staged child lists.
struct TreeSmem {
    unsigned long long* qkey;
    float* qps;
    int *qrow, *qrank, *qtok;
    int *o_tok, *o_par, *o_dep;
    float* o_score;
    int* topm;        // [gamma, M]
    uint32_t* anc;    // with the fused mask: [B + 1][(B + 32) / 32] ancestor-or-self bits
    uint8_t* lists;   // staged prefixes: ids [rows][sw] int32, then log-probs [rows][sw] float
};
__device__ __forceinline__ TreeSmem tree_smem(uint8_t* base, const TreeArgs& a) {
    TreeSmem t;
    const int cap = a.B + 2, n_out = a.B + 1;
    t.qkey = reinterpret_cast<unsigned long long*>(base);
    t.qps = reinterpret_cast<float*>(t.qkey + cap);
    t.qrow = reinterpret_cast<int*>(t.qps + cap);
    t.qrank = t.qrow + cap;
    t.qtok = t.qrank + cap;
    t.o_tok = t.qtok + cap;
    t.o_par = t.o_tok + n_out;
    t.o_dep = t.o_par + n_out;
    t.o_score = reinterpret_cast<float*>(t.o_dep + n_out);
    t.topm = reinterpret_cast<int*>(t.o_score + n_out);
    uint8_t* next = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(t.topm + a.gamma * a.M) + 15) &
                                               ~static_cast<uintptr_t>(15));
    t.anc = reinterpret_cast<uint32_t*>(next);
    if (a.mask)
        next = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(t.anc + tree_mask_words(n_out)) + 15) &
                                          ~static_cast<uintptr_t>(15));
    t.lists = next;
    return t;
}

// Stage sequence s's stage-1 top-M and the first sw entries of each of its child lists.
__device__ __forceinline__ ListView stage_sequence(const TreeArgs& a, int s, const TreeSmem& t, int sw) {
    const int tid = threadIdx.x;
    const bool ar = a.mode == TF_MODE_AR;
    const int n_rows_l = ar ? a.R : a.gamma;
    const int stride = ar ? a.K2 : a.K1;
    ListView v;
    v.g_ids = ar ? a.child_ids + static_cast<size_t>(s) * a.R * a.K2 : a.top_ids + static_cast<size_t>(s) * a.gamma * a.K1;
    v.g_lp = ar ? a.child_logp + static_cast<size_t>(s) * a.R * a.K2 : a.top_logp + static_cast<size_t>(s) * a.gamma * a.K1;
    v.stride = stride;
    v.sw = sw;
    for (int i = tid; i < a.gamma * a.M; i += kTreeThreads)
        t.topm[i] = a.top_ids[(static_cast<size_t>(s) * a.gamma + i / a.M) * a.K1 + i % a.M];
    const int n = n_rows_l * sw;
    int32_t* si = reinterpret_cast<int32_t*>(t.lists);
    float* sl = reinterpret_cast<float*>(si + n);
    v.s_ids = si;
    v.s_lp = sl;
    const bool vec = sw == stride &&
                     ((reinterpret_cast<uintptr_t>(v.g_ids) | reinterpret_cast<uintptr_t>(v.g_lp) |
                       reinterpret_cast<uintptr_t>(si) | reinterpret_cast<uintptr_t>(sl)) & 15) == 0 &&
                     (n & 3) == 0;
    constexpr int T = kTreeThreads;
    if (vec) {
        // whole lists: 16-byte copies, sixteen per thread in flight before the first store
        const int4* gi = reinterpret_cast<const int4*>(v.g_ids);
        const float4* gl = reinterpret_cast<const float4*>(v.g_lp);
        int4* di = reinterpret_cast<int4*>(si);
        float4* dl = reinterpret_cast<float4*>(sl);
        const int n4 = n >> 2;
        for (int base = tid; base < n4; base += 8 * T) {
            int4 va[8];
            float4 vb[8];
#pragma unroll
            for (int j = 0; j < 8; ++j)
                if (base + j * T < n4) {
                    va[j] = gi[base + j * T];
                    vb[j] = gl[base + j * T];
                }
#pragma unroll
            for (int j = 0; j < 8; ++j)
                if (base + j * T < n4) {
                    di[base + j * T] = va[j];
                    dl[base + j * T] = vb[j];
                }
        }
    } else {
        // prefixes of sw entries: element copies, eight per thread in flight
        for (int base = tid; base < n; base += 8 * T) {
            int32_t va[8];
            float vb[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int i = base + j * T;
                if (i < n) {
                    const size_t g = static_cast<size_t>(i / sw) * stride + i % sw;
                    va[j] = v.g_ids[g];
                    vb[j] = v.g_lp[g];
                }
            }
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int i = base + j * T;
                if (i < n) {
                    si[i] = va[j];
                    sl[i] = vb[j];
                }
            }
        }
    }
    return v;
}

// Nodes from shared memory to the outputs.
__device__ __forceinline__ void write_nodes(const TreeArgs& a, int s, const TreeSmem& t) {
    const int n_out = a.B + 1;
    for (int i = threadIdx.x; i < n_out; i += kTreeThreads) {
        const size_t o = static_cast<size_t>(s) * n_out + i;
        a.node_tok[o] = t.o_tok[i];
        a.node_parent[o] = t.o_par[i];
        a.node_depth[o] = t.o_dep[i];
        a.node_score[o] = t.o_score[i];
    }
}

// Rows r0 .. r1-1 of one sequence's tree-attention mask and their position ids. mask[i][j] = 1
// iff node j is node i or one of its ancestors; pos = root_pos + depth. Each node walks its own
// parent chain (at most kMaxGamma links) and sets the bits of its row, so no thread waits for
// another level. A node is present iff every link of its chain goes to a smaller index exactly
// one level up and the chain ends at the root (node 0, depth 0); absent nodes (missing from an
// underfull tree, or behind a broken link) get an empty row and column and pos -1.
// par, dep: the tree's n parents and depths (shared memory); anc: (r1 - r0) x W words of shared
// scratch; mask_s [n][n] and pos_s [n]: this sequence's outputs.
__device__ __forceinline__ void mask_rows(int n, const int* par, const int* dep, int root_pos, int r0, int r1,
                                          uint32_t* anc, uint8_t* mask_s, int32_t* pos_s) {
    const int W = (n + 31) / 32;
    for (int i = r0 + static_cast<int>(threadIdx.x); i < r1; i += blockDim.x) {
        uint32_t* row = anc + static_cast<size_t>(i - r0) * W;
        for (int w = 0; w < W; ++w) row[w] = 0u;
        bool ok = true;
        int j = i;
        for (int steps = 0; ok && j != 0; ++steps) {
            const int p = par[j];
            ok = steps < kMaxGamma && dep[j] >= 1 && dep[j] <= kMaxGamma && p >= 0 && p < j && dep[p] == dep[j] - 1;
            row[j >> 5] |= 1u << (j & 31);
            j = p;
        }
        ok = ok && dep[0] == 0;
        if (ok) {
            row[0] |= 1u;                                  // the root
        } else {
            for (int w = 0; w < W; ++w) row[w] = 0u;       // absent: empty row
        }
        pos_s[i] = ok ? root_pos + dep[i] : -1;
    }
    __syncthreads();
    const int count = (r1 - r0) * n;
    for (int idx = threadIdx.x; idx < count; idx += blockDim.x) {
        const int i = idx / n, jcol = idx - (idx / n) * n;
        mask_s[static_cast<size_t>(r0 + i) * n + jcol] = static_cast<uint8_t>((anc[i * W + (jcol >> 5)] >> (jcol & 31)) & 1u);
    }
}

// The fused mask of a builder CTA, once its tree is complete in shared memory.
__device__ __forceinline__ void fused_mask(const TreeArgs& a, int s, const TreeSmem& t) {
    if (!a.mask) return;
    const int n = a.B + 1;
    mask_rows(n, t.o_par, t.o_dep, a.root_pos[s], 0, n, t.anc, a.mask + static_cast<size_t>(s) * n * n,
              a.pos_ids + static_cast<size_t>(s) * n);
}

// General builder (any B): the queue in shared memory.
__global__ void __launch_bounds__(kTreeThreads) build_tree_kernel(TreeArgs a, int sw) {
    pdl_trigger();
    pdl_wait();
    extern __shared__ __align__(16) uint8_t smem_raw[];
    const TreeSmem t = tree_smem(smem_raw, a);
    unsigned long long* qkey = t.qkey;
    float* qps = t.qps;
    int* qrow = t.qrow;
    int* qrank = t.qrank;
    int* qtok = t.qtok;
    int* o_tok = t.o_tok;
    int* o_par = t.o_par;
    int* o_dep = t.o_dep;
    float* o_score = t.o_score;
    int* topm = t.topm;
    const int n_out = a.B + 1;
    const int s = blockIdx.x;
    const int tid = threadIdx.x;
    const bool ar = a.mode == TF_MODE_AR;
    const ListView lv = stage_sequence(a, s, t, sw);
    __syncthreads();

    if (tid < 32) {
        const int lane = tid;
        constexpr unsigned kFull = 0xffffffffu;
        int flags = 0;
        const int root = a.root_tok[a.two_prev ? 2 * s : s];
        if (root < 0 || root >= a.V) flags |= TF_DEV_BAD_TOKEN;
        const int list_len = a.K2;
        if (lane == 0) {
            o_tok[0] = root;
            o_par[0] = -1;
            o_dep[0] = 0;
            o_score[0] = 0.0f;
            qkey[0] = queue_key(lv.lp(0, 0), 1, 0);
            qps[0] = 0.0f;
            qrow[0] = 0;
            qrank[0] = 0;
            qtok[0] = lv.tok(0, 0);
        }
        int n_e = 1;
        int count = 1;
        __syncwarp();
        unsigned long long lbest = 0ull;
        int lidx = -1;
        auto rescan = [&]() {
            lbest = 0ull;
            lidx = -1;
            for (int j = lane; j < n_e; j += 32) {
                const unsigned long long k = qkey[j];
                if (k > lbest) {
                    lbest = k;
                    lidx = j;
                }
            }
        };
        rescan();
        while (count < n_out && n_e > 0) {
            const uint32_t hi = static_cast<uint32_t>(lbest >> 32), lo = static_cast<uint32_t>(lbest);
            const uint32_t mhi = __reduce_max_sync(kFull, hi);
            const uint32_t mlo = __reduce_max_sync(kFull, hi == mhi ? lo : 0u);
            const unsigned win = __ballot_sync(kFull, lbest != 0ull && hi == mhi && lo == mlo);
            if (win == 0u) break;
            const int best = __shfl_sync(kFull, lidx, __ffs(win) - 1);
            const float sc = key_float(mhi);
            const int dep = 127 - static_cast<int>(mlo >> 24);
            const int par = 0xFFFFFF - static_cast<int>(mlo & 0xFFFFFFu);
            const int row = qrow[best], rank = qrank[best], tok = qtok[best];
            const float psc = qps[best];
            __syncwarp();
            const int node = count++;
            if (tok < 0 || tok >= a.V) flags |= TF_DEV_BAD_TOKEN;
            if (!isfinite(sc)) flags |= TF_DEV_NONFINITE;
            // expandable? (depth cap; M-ary rule)
            int crow = -1;
            if (dep < a.gamma) {
                if (a.mode == TF_MODE_MARGINAL) {
                    crow = dep;
                } else {
                    const int m = mary_index(topm, dep, a.M, tok, lane, true);
                    if (m >= 0) crow = ar ? 1 + (dep - 1) * a.M + m : dep;
                    if (ar && a.two_prev) crow = child_row_2prev(topm, o_tok, a.M, dep, m, par, lane);
                }
            }
            const bool sibling = rank + 1 < list_len;
            const int last = n_e - 1;
            if (lane == 0) {
                o_tok[node] = tok;
                o_par[node] = par;
                o_dep[node] = dep;
                o_score[node] = sc;
                if (sibling) {                   // next sibling of the popped entry
                    qrank[best] = rank + 1;
                    qtok[best] = lv.tok(row, rank + 1);
                    qkey[best] = queue_key(psc + lv.lp(row, rank + 1), dep, par);
                } else if (best != last) {       // list exhausted: move the last entry here
                    qkey[best] = qkey[last];
                    qps[best] = qps[last];
                    qrow[best] = qrow[last];
                    qrank[best] = qrank[last];
                    qtok[best] = qtok[last];
                }
            }
            if (!sibling) --n_e;
            int fresh = -1;
            if (crow >= 0) {
                fresh = n_e;
                if (lane == 0) {
                    qkey[n_e] = queue_key(sc + lv.lp(crow, 0), dep + 1, node);
                    qps[n_e] = sc;
                    qrow[n_e] = crow;
                    qrank[n_e] = 0;
                    qtok[n_e] = lv.tok(crow, 0);
                }
                ++n_e;
            }
            __syncwarp();
            if (lane == (best & 31) || (!sibling && lane == (last & 31)) || (fresh >= 0 && lane == (fresh & 31)))
                rescan();
        }
        if (count < n_out) flags |= TF_DEV_UNDERFULL;
        for (int i = count + lane; i < n_out; i += 32) {
            o_tok[i] = -1;
            o_par[i] = -1;
            o_dep[i] = -1;
            o_score[i] = -INFINITY;
        }
        if (lane == 0) a.dev_status[s] = sequence_status(a, flags);
    }
    __syncthreads();
    write_nodes(a, s, t);
    fused_mask(a, s, t);
}

// Builder for B + 1 <= 32 S: the queue in registers, S slots per lane (slot j on lane j % 32,
// register j / 32). Slots are appended in pop order and an exhausted list leaves an empty slot
// (key 0, below every real key), so no entry ever moves. Pops, tie rules and results are those
// of build_tree_kernel.
template <int S, bool FULL>
__global__ void __launch_bounds__(kTreeThreads) build_tree_reg_kernel(TreeArgs a, int sw) {
    pdl_trigger();
    pdl_wait();
    extern __shared__ __align__(16) uint8_t smem_raw[];
    const TreeSmem t = tree_smem(smem_raw, a);
    const int n_out = a.B + 1;
    const int s = blockIdx.x;
    const bool ar = a.mode == TF_MODE_AR;
    const ListView lv = stage_sequence(a, s, t, sw);
    // FULL: every rank a pop can reach is staged, so entries are read from shared memory only
    auto ltok = [&](int row, int rank) { return FULL ? lv.s_ids[row * sw + rank] : lv.tok(row, rank); };
    auto llp = [&](int row, int rank) { return FULL ? lv.s_lp[row * sw + rank] : lv.lp(row, rank); };
    __syncthreads();
    if (threadIdx.x < 32) {
        const int lane = threadIdx.x;
        constexpr unsigned kFull = 0xffffffffu;
        int flags = 0;
        const int root = a.root_tok[a.two_prev ? 2 * s : s];
        if (root < 0 || root >= a.V) flags |= TF_DEV_BAD_TOKEN;
        const int list_len = a.K2;
        unsigned long long key[S];
        int srow[S], srank[S], stok[S];
        float spsc[S];
#pragma unroll
        for (int j = 0; j < S; ++j) {
            key[j] = 0ull;
            srow[j] = srank[j] = stok[j] = 0;
            spsc[j] = 0.0f;
        }
        if (lane == 0) {
            key[0] = queue_key(llp(0, 0), 1, 0);
            stok[0] = ltok(0, 0);
            t.o_tok[0] = root;
            t.o_par[0] = -1;
            t.o_dep[0] = 0;
            t.o_score[0] = 0.0f;
        }
        int n_e = 1;      // slots used so far
        int count = 1;    // nodes placed
        while (count < n_out) {
            // this lane's best slot and its entry
            unsigned long long lb = key[0];
            int brow = srow[0], brank = srank[0], btok = stok[0];
            float bpsc = spsc[0];
#pragma unroll
            for (int j = 1; j < S; ++j)
                if (key[j] > lb) {
                    lb = key[j];
                    brow = srow[j];
                    brank = srank[j];
                    btok = stok[j];
                    bpsc = spsc[j];
                }
            const uint32_t hi = static_cast<uint32_t>(lb >> 32), lo = static_cast<uint32_t>(lb);
            const uint32_t mhi = __reduce_max_sync(kFull, hi);
            if (mhi == 0u) break;                      // queue empty (every real key has hi > 0)
            unsigned win = __ballot_sync(kFull, hi == mhi);
            if (__popc(win) > 1) {
                const uint32_t mlo = __reduce_max_sync(kFull, hi == mhi ? lo : 0u);
                win = __ballot_sync(kFull, hi == mhi && lo == mlo);
            }
            const int wl = __ffs(win) - 1;
            const uint32_t wlo = __shfl_sync(kFull, lo, wl);
            const int row = __shfl_sync(kFull, brow, wl);
            const int rank = __shfl_sync(kFull, brank, wl);
            const int tok = __shfl_sync(kFull, btok, wl);
            const float psc = __shfl_sync(kFull, bpsc, wl);
            const float sc = key_float(mhi);
            const int dep = 127 - static_cast<int>(wlo >> 24);
            const int par = 0xFFFFFF - static_cast<int>(wlo & 0xFFFFFFu);
            const int node = count++;
            // next sibling of the popped entry (the same shared-memory words for every lane),
            // read before the expandability test so that both latencies overlap
            const bool sibling = rank + 1 < list_len;
            const int sib_tok = sibling ? ltok(row, rank + 1) : 0;
            const float sib_lp = sibling ? llp(row, rank + 1) : 0.0f;
            // expandable? (depth cap; M-ary rule)
            const bool deep_ok = dep < a.gamma;
            const int m = mary_index(t.topm, dep, a.M, tok, lane, deep_ok && a.mode != TF_MODE_MARGINAL);
            int crow = !deep_ok ? -1
                       : a.mode == TF_MODE_MARGINAL ? dep
                       : m >= 0 ? (ar ? 1 + (dep - 1) * a.M + m : dep) : -1;
            if (ar && a.two_prev) crow = child_row_2prev(t.topm, t.o_tok, a.M, dep, deep_ok ? m : -1, par, lane);
            if (tok < 0 || tok >= a.V) flags |= TF_DEV_BAD_TOKEN;
            if (!isfinite(sc)) flags |= TF_DEV_NONFINITE;
            const unsigned long long sib_key = sibling ? queue_key(psc + sib_lp, dep, par) : 0ull;
            if (lane == wl) {
                // the winner's best slot is the one holding its best key (keys are unique)
#pragma unroll
                for (int j = 0; j < S; ++j) {
                    const bool m = key[j] == lb;
                    key[j] = m ? sib_key : key[j];
                    srank[j] = m ? rank + 1 : srank[j];
                    stok[j] = m ? sib_tok : stok[j];
                }
            }
            if (crow >= 0) {
                const int ctok = ltok(crow, 0);
                const unsigned long long ckey = queue_key(sc + llp(crow, 0), dep + 1, node);
                const bool mine = lane == (n_e & 31);
#pragma unroll
                for (int j = 0; j < S; ++j) {
                    const bool m = mine && j == (n_e >> 5);
                    key[j] = m ? ckey : key[j];
                    srow[j] = m ? crow : srow[j];
                    srank[j] = m ? 0 : srank[j];
                    stok[j] = m ? ctok : stok[j];
                    spsc[j] = m ? sc : spsc[j];
                }
                ++n_e;
            }
            if (lane == 0) {
                t.o_tok[node] = tok;
                t.o_par[node] = par;
                t.o_dep[node] = dep;
                t.o_score[node] = sc;
            }
        }
        if (count < n_out) flags |= TF_DEV_UNDERFULL;
        for (int i = count + lane; i < n_out; i += 32) {
            t.o_tok[i] = -1;
            t.o_par[i] = -1;
            t.o_dep[i] = -1;
            t.o_score[i] = -INFINITY;
        }
        if (lane == 0) a.dev_status[s] = sequence_status(a, flags);
    }
    __syncthreads();
    write_nodes(a, s, t);
    fused_mask(a, s, t);
}

// ------------------------------------------------------------------------------------------
// Builder with a sorted queue, for the one-token rule and the marginal modes with B <= 64 and
// every reachable list entry staged. The same pops, tie rules and results as
// build_tree_reg_kernel. After t pops only the B - t best live entries can still be popped (each
// needs every better entry popped first), and at most t + 1 entries are live (a pop replaces its
// entry by the next sibling and adds at most the node's first child), so at most
// min(t + 1, B - t) <= 32 entries matter: lane i of one warp holds the i-th best. A pop takes
// lane 0's entry, tests its token against the stage-1 candidates of its depth with a ballot
// (the M-ary rule), and places its two successors (next sibling, first child) with two ballots
// over the remaining keys; every lane then takes its new entry from itself or a neighbour by
// shuffle. There is no warp-wide max and no divergent branch. The queue carries keys and list
// entries only (a sibling's parent score is the placed parent's o_score); a pop costs about
// 250 ns on GB300, a chain of about a hundred dependent single-warp instructions.
// ------------------------------------------------------------------------------------------
constexpr int kFastThreads = 512;
// Shared-memory bytes of build_tree_fast_kernel: nodes, candidates, mask bits and the staged
// lists (token and log-probability of every entry).
__host__ __device__ inline size_t fast_tree_smem(int B, int gamma, int M, int rows, int sw, bool with_mask) {
    const size_t n = static_cast<size_t>(B) + 1;
    size_t bytes = n * 16 + static_cast<size_t>(gamma) * M * 4;
    bytes = (bytes + 15) & ~static_cast<size_t>(15);
    if (with_mask) bytes += (tree_mask_words(static_cast<int>(n)) * 4 + 15) & ~static_cast<size_t>(15);
    return bytes + static_cast<size_t>(rows) * sw * 8 + 16;
}

__device__ __forceinline__ bool key_gt(uint32_t ahi, uint32_t alo, uint32_t bhi, uint32_t blo) {
    return ahi > bhi || (ahi == bhi && alo > blo);
}

__global__ void __launch_bounds__(kFastThreads) build_tree_fast_kernel(TreeArgs a, int sw) {
    pdl_trigger();
    pdl_wait();
    extern __shared__ __align__(16) uint8_t smem_raw[];
    constexpr unsigned kFull = 0xffffffffu;
    const int n_out = a.B + 1, s = blockIdx.x, tid = threadIdx.x;
    const int T = blockDim.x;
    const bool ar = a.mode == TF_MODE_AR, mary = a.mode != TF_MODE_MARGINAL;
    const int rows_l = ar ? a.R : a.gamma;
    const int stride = ar ? a.K2 : a.K1;
    // every array is carved by a byte offset into smem_raw, so that all accesses stay
    // shared-memory accesses
    int* o_tok = reinterpret_cast<int*>(smem_raw);
    int* o_par = o_tok + n_out;
    int* o_dep = o_par + n_out;
    float* o_score = reinterpret_cast<float*>(o_dep + n_out);
    int* topm = reinterpret_cast<int*>(o_score + n_out);
    size_t off = (static_cast<size_t>(reinterpret_cast<uint8_t*>(topm + a.gamma * a.M) - smem_raw) + 15) & ~static_cast<size_t>(15);
    uint32_t* anc = reinterpret_cast<uint32_t*>(smem_raw + off);
    if (a.mask) off += (tree_mask_words(n_out) * 4 + 15) & ~static_cast<size_t>(15);
    const int n = rows_l * sw;
    int* l_tok = reinterpret_cast<int*>(smem_raw + off);
    float* l_lp = reinterpret_cast<float*>(l_tok + n);

    // ---- the lists and the stage-1 candidates
    const int32_t* g_ids = ar ? a.child_ids + static_cast<size_t>(s) * a.R * a.K2
                              : a.top_ids + static_cast<size_t>(s) * a.gamma * a.K1;
    const float* g_lp = ar ? a.child_logp + static_cast<size_t>(s) * a.R * a.K2
                           : a.top_logp + static_cast<size_t>(s) * a.gamma * a.K1;
    const bool vec = sw == stride && (sw & 3) == 0 &&
                     ((reinterpret_cast<uintptr_t>(g_ids) | reinterpret_cast<uintptr_t>(g_lp)) & 15) == 0;
    if (vec) {
        const int n4 = n >> 2;
        const int4* gi = reinterpret_cast<const int4*>(g_ids);
        const float4* gl = reinterpret_cast<const float4*>(g_lp);
        for (int base = tid; base < n4; base += 8 * T) {
            int4 vi[8];
            float4 vl[8];
#pragma unroll
            for (int u = 0; u < 8; ++u)
                if (base + u * T < n4) {
                    vi[u] = gi[base + u * T];
                    vl[u] = gl[base + u * T];
                }
#pragma unroll
            for (int u = 0; u < 8; ++u)
                if (base + u * T < n4) {
                    reinterpret_cast<int4*>(l_tok)[base + u * T] = vi[u];
                    reinterpret_cast<float4*>(l_lp)[base + u * T] = vl[u];
                }
        }
    } else {
        for (int i = tid; i < n; i += T) {
            const int r = i / sw;
            const size_t g = static_cast<size_t>(r) * stride + (i - r * sw);
            l_tok[i] = g_ids[g];
            l_lp[i] = g_lp[g];
        }
    }
    for (int i = tid; i < a.gamma * a.M; i += T)
        topm[i] = a.top_ids[(static_cast<size_t>(s) * a.gamma + i / a.M) * a.K1 + i % a.M];
    __syncthreads();
    // ---- the pops (one warp): lane i holds the i-th best live entry, as its key (score, depth,
    // parent) and its list entry (row << 10 | rank); key 0 marks an empty lane. The parent's
    // score, which a sibling's score needs, is read from the placed nodes (o_score[parent]).
    if (tid < 32) {
        const int lane = tid;
        const int list_len = a.K2 < sw ? a.K2 : sw;   // staged ranks; a pop never reaches rank sw
        int flags = 0;
        const int root = a.root_tok[s];
        if (root < 0 || root >= a.V) flags |= TF_DEV_BAD_TOKEN;
        uint32_t khi = 0u, klo = 0u;
        int rr = 0;
        if (lane == 0) {
            const unsigned long long k0 = queue_key(l_lp[0], 1, 0);
            khi = static_cast<uint32_t>(k0 >> 32);
            klo = static_cast<uint32_t>(k0);
            o_tok[0] = root;
            o_par[0] = -1;
            o_dep[0] = 0;
            o_score[0] = 0.0f;
        }
        int count = 1;    // nodes placed
        while (count < n_out) {
            __syncwarp();                              // lane 0's node writes, for o_score below
            // the head: lane 0's entry
            const uint32_t hhi = __shfl_sync(kFull, khi, 0);
            if (hhi == 0u) break;                      // queue empty
            const uint32_t hlo = __shfl_sync(kFull, klo, 0);
            const int hrr = __shfl_sync(kFull, rr, 0);
            // the rest shifted by one: lane i sees entries i + 1 (next) and i - 1 (prev)
            uint32_t nhi = __shfl_down_sync(kFull, khi, 1), nlo = __shfl_down_sync(kFull, klo, 1);
            const int nrr = __shfl_down_sync(kFull, rr, 1);
            if (lane == 31) nhi = nlo = 0u;
            const uint32_t phi = __shfl_up_sync(kFull, khi, 1), plo = __shfl_up_sync(kFull, klo, 1);
            const int prr = __shfl_up_sync(kFull, rr, 1);
            // the popped node
            const int row = hrr >> 10, rank = hrr & 1023, idx = row * sw + rank;
            const int dep = 127 - static_cast<int>(hlo >> 24);
            const int par = 0xFFFFFF - static_cast<int>(hlo & 0xFFFFFFu);
            const float sc = key_float(hhi);
            const int node = count++;
            const int tok = l_tok[idx];
            const float hpsc = o_score[par];           // the parent's score
            // its children: none at the depth cap; DDTree: the next depth's marginal row;
            // otherwise only for a stage-1 candidate m of its depth (Algorithm 1 Part 2), found by
            // ballots over the depth's candidates (the first equal one counts): stage-2 row
            // 1 + (dep - 1) M + m, or the next marginal row
            const int* cand = topm + (dep < a.gamma && mary ? (dep - 1) * a.M : 0);
            const int c0 = lane < a.M ? cand[lane] : -1;
            const unsigned b0 = __ballot_sync(kFull, lane < a.M && c0 == tok);
            int m = b0 ? __ffs(b0) - 1 : -1;
            if (a.M > 32) {                            // (the same for every lane)
                const int c1 = lane + 32 < a.M ? cand[lane + 32] : -1;
                const unsigned b1 = __ballot_sync(kFull, lane + 32 < a.M && c1 == tok);
                m = b0 ? m : b1 ? 32 + __ffs(b1) - 1 : -1;
            }
            const int crow = dep >= a.gamma ? -1 : !mary ? dep : m < 0 ? -1 : ar ? 1 + (dep - 1) * a.M + m : dep;
            const bool sib_ok = rank + 1 < list_len;
            const float slp = l_lp[sib_ok ? idx + 1 : idx];
            const bool ch_ok = crow >= 0 && node + 1 < n_out;   // nothing is popped after the last node
            const float clp = l_lp[ch_ok ? crow * sw : 0];
            if (lane == 0) {
                if (tok < 0 || tok >= a.V) flags |= TF_DEV_BAD_TOKEN;
                if (!isfinite(sc)) flags |= TF_DEV_NONFINITE;
                o_tok[node] = tok;
                o_par[node] = par;
                o_dep[node] = dep;
                o_score[node] = sc;
            }
            // its successors, A before B in queue order (0 = none): the next sibling shares the
            // head's depth and parent (the low word of its key), the child is one level deeper
            // with this node as parent
            const uint32_t shi = sib_ok ? float_key(hpsc + slp) : 0u, slo = sib_ok ? hlo : 0u;
            const uint32_t chi = ch_ok ? float_key(sc + clp) : 0u;
            const uint32_t clo = ch_ok ? (static_cast<uint32_t>(126 - dep) << 24) | static_cast<uint32_t>(0xFFFFFF - node) : 0u;
            const bool s_first = key_gt(shi, slo, chi, clo);
            const uint32_t ahi = s_first ? shi : chi, alo = s_first ? slo : clo;
            const uint32_t bhi = s_first ? chi : shi, blo = s_first ? clo : slo;
            const int arr = s_first ? hrr + 1 : crow << 10, brr = s_first ? crow << 10 : hrr + 1;
            // their places among the remaining entries (sorted, so the larger keys are a prefix)
            const int pA = __popc(__ballot_sync(kFull, key_gt(nhi, nlo, ahi, alo)));
            const int pB = __popc(__ballot_sync(kFull, key_gt(nhi, nlo, bhi, blo)));
            // new entry i: rest[i] before A, A, rest[i - 1] up to B, B, rest[i - 2] after it
            const int j = lane;
            const bool takeA = j == pA, takeB = j == pB + 1;
            const bool fromN = j < pA, fromO = j > pA && j <= pB;
            khi = takeA ? ahi : takeB ? bhi : fromN ? nhi : fromO ? khi : phi;
            klo = takeA ? alo : takeB ? blo : fromN ? nlo : fromO ? klo : plo;
            rr = takeA ? arr : takeB ? brr : fromN ? nrr : fromO ? rr : prr;
        }
        flags = static_cast<int>(__reduce_or_sync(kFull, static_cast<unsigned>(flags)));
        if (count < n_out) flags |= TF_DEV_UNDERFULL;
        for (int i = count + lane; i < n_out; i += 32) {
            o_tok[i] = -1;
            o_par[i] = -1;
            o_dep[i] = -1;
            o_score[i] = -INFINITY;
        }
        if (lane == 0) a.dev_status[s] = sequence_status(a, flags);
    }
    __syncthreads();
    for (int i = tid; i < n_out; i += T) {
        const size_t o = static_cast<size_t>(s) * n_out + i;
        a.node_tok[o] = o_tok[i];
        a.node_parent[o] = o_par[i];
        a.node_depth[o] = o_dep[i];
        a.node_score[o] = o_score[i];
    }
    if (a.mask)
        mask_rows(n_out, o_par, o_dep, a.root_pos[s], 0, n_out, anc, a.mask + static_cast<size_t>(s) * n_out * n_out,
                  a.pos_ids + static_cast<size_t>(s) * n_out);
}

// ------------------------------------------------------------------------------------------
// The tree-attention mask and position ids (mask_rows) of a drafted tree in global memory: one
// CTA per sequence and block of kMaskRows rows.
// ------------------------------------------------------------------------------------------
__global__ void __launch_bounds__(256) tree_mask_kernel(int n, const int32_t* __restrict__ node_parent,
                                                        const int32_t* __restrict__ node_depth,
                                                        const int32_t* __restrict__ root_pos,
                                                        uint8_t* __restrict__ mask, int32_t* __restrict__ pos_ids) {
    pdl_trigger();
    pdl_wait();
    extern __shared__ uint32_t sm[];
    const int s = blockIdx.x;
    const int r0 = blockIdx.y * kMaskRows, r1 = min(n, r0 + kMaskRows);   // this CTA's rows
    int* par = reinterpret_cast<int*>(sm);
    int* dep = par + n;
    uint32_t* anc = reinterpret_cast<uint32_t*>(dep + n);   // [kMaskRows][(n + 31) / 32] ancestor-or-self bits
    const int32_t* P = node_parent + static_cast<size_t>(s) * n;
    const int32_t* D = node_depth + static_cast<size_t>(s) * n;
    for (int i = threadIdx.x; i < n; i += blockDim.x) {
        par[i] = P[i];
        dep[i] = D[i];
    }
    __syncthreads();
    mask_rows(n, par, dep, root_pos[s], r0, r1, anc, mask + static_cast<size_t>(s) * n * n,
              pos_ids + static_cast<size_t>(s) * n);
}

// ------------------------------------------------------------------------------------------
// Verification walk (Sec. 3: a drafted token is accepted iff it equals the verifier's token at
// its parent's position; Sec. 4: the step gains the accepted tokens plus the verifier's residual
// token). One warp per sequence: from the root, each step finds the child of the current node
// whose token equals the verifier's token there (a ballot over all nodes; the smallest index if
// an invalid tree repeats a token) and moves to it. At most gamma steps (the depth cap), so a
// corrupt parent array cannot loop.
// ------------------------------------------------------------------------------------------
__global__ void __launch_bounds__(32) accept_walk_kernel(int n, int gamma, const int32_t* __restrict__ node_tok,
                                                         const int32_t* __restrict__ node_parent,
                                                         const int32_t* __restrict__ verifier_tok,
                                                         int32_t* __restrict__ accept_len,
                                                         int32_t* __restrict__ accept_path,
                                                         int32_t* __restrict__ next_tok) {
    pdl_trigger();
    pdl_wait();
    constexpr unsigned kFull = 0xffffffffu;
    const int s = blockIdx.x, lane = threadIdx.x;
    const int32_t* tok = node_tok + static_cast<size_t>(s) * n;
    const int32_t* par = node_parent + static_cast<size_t>(s) * n;
    const int32_t* ver = verifier_tok + static_cast<size_t>(s) * n;
    int32_t* path = accept_path + static_cast<size_t>(s) * (gamma + 1);
    int cur = 0, len = 0;
    if (lane == 0) path[0] = 0;
    for (int step = 0; step < gamma; ++step) {
        const int want = ver[cur];
        int found = -1;
        for (int c0 = 1; c0 < n && found < 0; c0 += 32) {
            const int c = c0 + lane;
            const bool m = c < n && par[c] == cur && tok[c] == want;
            const unsigned bal = __ballot_sync(kFull, m);
            if (bal) found = c0 + __ffs(bal) - 1;
        }
        if (found < 0) break;
        cur = found;
        ++len;
        if (lane == 0) path[len] = cur;
    }
    for (int i = len + 1 + lane; i <= gamma; i += 32) path[i] = -1;
    if (lane == 0) {
        accept_len[s] = len;
        next_tok[s] = ver[cur];
    }
}

}  // namespace

// Error-free sum (Knuth's TwoSum): s + c tracks a running sum to about twice fp32 precision.
__device__ __forceinline__ void two_sum_acc(float& s, float& c, float x) {
    const float t = s + x;
    const float z = t - s;
    c += (s - (t - z)) + (x - z);
    s = t;
}

// bf16 nearest-even rounding of the real value r + t, where r is an fp32 value and |t| is below
// two fp32 ulps of r. Only an r within a few ulps of a bf16 midpoint can round differently from
// r alone; for those the side of the midpoint is decided from (r - midpoint) + t, where
// r - midpoint is exact (both share r's binade).
__device__ __forceinline__ __nv_bfloat16 bf16_round_sum(float r, float t) {
    const uint32_t u = __float_as_uint(r);
    const uint32_t low = u & 0xffffu;
    if ((u & 0x7f800000u) == 0x7f800000u || low < 0x8000u - 4u || low > 0x8000u + 4u) return __float2bfloat16_rn(r);
    const uint32_t trunc = u & 0xffff0000u;
    const float mid = __uint_as_float(trunc | 0x8000u);
    const float dm = (r - mid) + t;
    const float away = (u & 0x80000000u) ? -dm : dm;   // > 0: beyond the midpoint in magnitude
    uint32_t bits = trunc;
    if (away > 0.0f || (away == 0.0f && (trunc & 0x10000u))) bits += 0x10000u;
    return __ushort_as_bfloat16(static_cast<unsigned short>(bits >> 16));
}

// bf16 rows with d % 8 == 0: 16-byte loads and stores, 8 elements per thread and step. x is the
// correctly rounded bf16 value of the definition (an element off by one bf16 ulp would perturb
// every gate/up output and flip many later roundings), computed in fp32 only (GB300's fp64 is too
// slow even for the few scalar steps of a row):
//  - mean(h^2): every square of a bf16 value is exact in fp32; the sums, and their warp and block
//    reductions, are compensated (TwoSum pairs);
//  - 1 / sqrt(mean + eps) as hi + lo: hi = rsqrtf, then one Newton step in double-float
//    arithmetic (the squares and products formed exactly with FMAs), about 2^-46 relative;
//  - h * w is exact in fp32 (two 8-bit significands); (h w) * hi is rounded once and its
//    rounding error recovered with an FMA, so (h w) / sqrt(mean + eps) is known as r + t to
//    about 2^-45 relative, which decides the bf16 rounding (bf16_round_sum).
template <int NE>
__global__ void __launch_bounds__(256) gather_norm_bf16x8_kernel(
    const uint4* __restrict__ hidden, const uint4* __restrict__ embed, const uint4* __restrict__ norm_h,
    const uint4* __restrict__ norm_e, const int32_t* __restrict__ root_tok, const int32_t* __restrict__ top_ids,
    int gamma, int M, int K1, int R, int d, int V, float eps, uint4* __restrict__ X, uint4* __restrict__ hres,
    int* status) {
    pdl_trigger();
    constexpr int kMaxPerThread = 4;          // d <= 256 * 8 * 4 = 8192
    constexpr int NS = 1 + NE;                // parts of x: the hidden state, then NE embeddings
    __shared__ float red[NS][2][8];
    __shared__ float scale[2 * NS];           // hi, lo of 1 / sqrt(mean + eps) of every part
    const int row = blockIdx.x;
    const int hid = stage2_row_hidden(row, R, gamma, M, NE == 2);

    const int dv = d / 8;
    // the hidden state and the norm weights are step inputs (no kernel writes them): read before
    // waiting for the previous kernel, which produces the candidate tokens
    const uint4* h = hidden + static_cast<size_t>(hid) * dv;
    uint4 v[NS][kMaxPerThread], wh[kMaxPerThread], we[kMaxPerThread];
#pragma unroll
    for (int i = 0; i < kMaxPerThread; ++i) {
        const int c = threadIdx.x + i * 256;
        if (c < dv) {
            v[0][i] = h[c];
            wh[i] = norm_h[c];
            we[i] = norm_e[c];
        }
    }
    pdl_wait();
    // the approximator GEMMs' tail-split counters (after the status word) start each call at zero
    if (blockIdx.x == 0 && status)
        for (int i = threadIdx.x; i < kTailSems; i += blockDim.x) status[1 + i] = 0;
    int tok[2] = {0, 0};
    stage2_row_tokens(row, R, gamma, M, K1, NE == 2, root_tok, top_ids, tok);
#pragma unroll
    for (int j = 0; j < NE; ++j) {
        if (tok[j] < 0 || tok[j] >= V) {
            if (threadIdx.x == 0) set_status(status, TF_DEV_BAD_TOKEN);
            tok[j] = 0;
        }
        const uint4* e = embed + static_cast<size_t>(tok[j]) * dv;
#pragma unroll
        for (int i = 0; i < kMaxPerThread; ++i) {
            const int c = threadIdx.x + i * 256;
            if (c < dv) v[1 + j][i] = e[c];
        }
    }
    // sums of squares: every square of a bf16 value is exact in fp32; the running sums are
    // compensated (TwoSum), and the (sum, compensation) pairs are combined the same way
    float sum[NS], comp[NS];
#pragma unroll
    for (int j = 0; j < NS; ++j) sum[j] = comp[j] = 0.0f;
#pragma unroll
    for (int i = 0; i < kMaxPerThread; ++i) {
        const int c = threadIdx.x + i * 256;
        if (c < dv) {
#pragma unroll
            for (int j = 0; j < NS; ++j) {
                const __nv_bfloat16* b = reinterpret_cast<const __nv_bfloat16*>(&v[j][i]);
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    const float a = __bfloat162float(b[k]);
                    two_sum_acc(sum[j], comp[j], a * a);
                }
            }
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
#pragma unroll
        for (int j = 0; j < NS; ++j) {
            const float s2 = __shfl_xor_sync(0xffffffffu, sum[j], o);
            const float c2 = __shfl_xor_sync(0xffffffffu, comp[j], o);
            two_sum_acc(sum[j], comp[j], s2);
            comp[j] += c2;
        }
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0)
#pragma unroll
        for (int j = 0; j < NS; ++j) {
            red[j][0][warp] = sum[j];
            red[j][1][warp] = comp[j];
        }
    __syncthreads();
    if (threadIdx.x < NS) {
        const int j = threadIdx.x;
        float S = 0.0f, C = 0.0f;
        for (int w = 0; w < 8; ++w) {
            two_sum_acc(S, C, red[j][0][w]);
            C += red[j][1][w];
        }
        // m = (S + C) / d + eps as a double-float (mh, ml); d is scaled exactly when it is a
        // power of two, otherwise the quotient's rounding error is recovered by an FMA
        const float fd = static_cast<float>(d);
        const float q = S / fd;
        const float qerr = fmaf(-q, fd, S) / fd + C / fd;
        float mh = q + eps;
        float ml = (q - (mh - (mh - q))) + (eps - (mh - q)) + qerr;   // TwoSum(q, eps) plus the rest
        const float t = mh + ml;
        ml = ml - (t - mh);
        mh = t;
        // y = 1 / sqrt(m): y0 = rsqrtf(mh), then one Newton step in double-float arithmetic,
        // y = y0 + y0 (1 - m y0^2) / 2, with y0^2 and m y0^2 formed by exact FMA products
        const float y0 = rsqrtf(mh);
        const float p = y0 * y0, pl = fmaf(y0, y0, -p);          // y0^2 = p + pl exactly
        const float u = mh * p, ul = fmaf(mh, p, -u);              // mh p = u + ul exactly
        const float r = ((1.0f - u) - ul) - (mh * pl + ml * p);    // 1 - m y0^2, ~2^-23
        const float hi = y0, lo = 0.5f * y0 * r;
        scale[2 * j] = hi;
        scale[2 * j + 1] = lo;
    }
    __syncthreads();
    uint4* xr = X + static_cast<size_t>(row) * NS * dv;
#pragma unroll
    for (int i = 0; i < kMaxPerThread; ++i) {
        const int c = threadIdx.x + i * 256;
        if (c < dv) {
#pragma unroll
            for (int j = 0; j < NS; ++j) {
                const float is = scale[2 * j], is_lo = scale[2 * j + 1];
                const __nv_bfloat16* b = reinterpret_cast<const __nv_bfloat16*>(&v[j][i]);
                const __nv_bfloat16* wb = reinterpret_cast<const __nv_bfloat16*>(j == 0 ? &wh[i] : &we[i]);
                uint4 o;
                __nv_bfloat16* ob = reinterpret_cast<__nv_bfloat16*>(&o);
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    const float pv = __bfloat162float(b[k]) * __bfloat162float(wb[k]);
                    const float rv = pv * is;
                    ob[k] = bf16_round_sum(rv, fmaf(pv, is_lo, fmaf(pv, is, -rv)));
                }
                xr[j * dv + c] = o;
            }
            if (NE == 2) hres[static_cast<size_t>(row) * dv + c] = v[0][i];
        }
    }
}

cudaError_t launch_gather_norm(const Ctx& ctx, int dtype, const void* hidden, const void* embed, const void* norm_h,
                               const void* norm_e, const int32_t* root_tok, const int32_t* top_ids, int b, int gamma,
                               int M, int K1, int R, int two_prev, int d, int V, float eps, void* X, void* hres) {
    const int rows = b * R;
    if (rows <= 0) return cudaSuccess;
    if (two_prev && !hres) return cudaErrorInvalidValue;
    cudaError_t e;
    if (dtype == TF_BF16 && d % 8 == 0 && d <= 8192) {
        auto kern = two_prev ? gather_norm_bf16x8_kernel<2> : gather_norm_bf16x8_kernel<1>;
        e = launch_pdl(kern, dim3(rows), dim3(256), 0, ctx.stream, static_cast<const uint4*>(hidden),
                       static_cast<const uint4*>(embed), static_cast<const uint4*>(norm_h),
                       static_cast<const uint4*>(norm_e), root_tok, top_ids, gamma, M, K1, R, d, V, eps,
                       static_cast<uint4*>(X), static_cast<uint4*>(hres), ctx.status);
    } else if (dtype == TF_BF16) {
        using B16 = __nv_bfloat16;
        auto kern = two_prev ? gather_norm_kernel<B16, 2> : gather_norm_kernel<B16, 1>;
        e = launch_pdl(kern, dim3(rows), dim3(256), 0, ctx.stream, static_cast<const B16*>(hidden),
                       static_cast<const B16*>(embed), static_cast<const B16*>(norm_h), static_cast<const B16*>(norm_e),
                       root_tok, top_ids, gamma, M, K1, R, d, V, eps, static_cast<B16*>(X), static_cast<B16*>(hres),
                       ctx.status);
    } else {
        auto kern = two_prev ? gather_norm_kernel<float, 2> : gather_norm_kernel<float, 1>;
        e = launch_pdl(kern, dim3(rows), dim3(256), 0, ctx.stream, static_cast<const float*>(hidden),
                       static_cast<const float*>(embed), static_cast<const float*>(norm_h),
                       static_cast<const float*>(norm_e), root_tok, top_ids, gamma, M, K1, R, d, V, eps,
                       static_cast<float*>(X), static_cast<float*>(hres), ctx.status);
    }
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t launch_build_tree(const Ctx& ctx, int b, int gamma, int M, int K1, int K2, int B, int V, int mode, int R,
                              int two_prev, const int32_t* root_tok, const int32_t* top_ids, const float* top_logp,
                              const int32_t* child_ids, const float* child_logp, int32_t* node_tok,
                              int32_t* node_parent, int32_t* node_depth, float* node_score, int32_t* dev_status,
                              const int32_t* root_pos, uint8_t* mask, int32_t* pos_ids, const int32_t* ws_status) {
    if (mask && B + 1 > kFusedMaskMaxNodes) return cudaErrorInvalidValue;
    TreeArgs a{gamma, M, K1, K2, B, V, mode, R, mode == TF_MODE_AR && two_prev ? 1 : 0, root_tok, top_ids, top_logp,
               child_ids, child_logp, node_tok, node_parent, node_depth, node_score, dev_status, root_pos, mask,
               pos_ids, ws_status};
    const size_t fixed = tree_smem_fixed(B, gamma, M, mask != nullptr);
    const int rows_l = mode == TF_MODE_AR ? R : gamma;
    const int stride = mode == TF_MODE_AR ? K2 : K1;
    // stage the entries a tree can reach (rank <= B) when they fit, else a prefix that does
    const int sw_full = stride < B + 1 ? stride : B + 1;
    int sw = sw_full;
    if (fixed + tree_smem_lists(rows_l, sw) > kTreeSmemLimit) {
        const size_t room = kTreeSmemLimit > fixed ? kTreeSmemLimit - fixed : 0;
        sw = static_cast<int>(room / (static_cast<size_t>(rows_l) * 8)) & ~3;
        if (sw > sw_full) sw = sw_full;
    }
    // the sorted-queue builder for the one-token rule and the marginal modes with B <= 64 and
    // every reachable entry staged
    if (!a.two_prev && B <= 64) {
        const size_t fsm = fast_tree_smem(B, gamma, M, rows_l, sw_full, mask != nullptr);
        if (fsm <= kTreeSmemLimit) {
            cudaError_t e = cudaFuncSetAttribute(build_tree_fast_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 static_cast<int>(fsm));
            if (e != cudaSuccess) return e;
            e = launch_pdl(build_tree_fast_kernel, dim3(b), dim3(kFastThreads), fsm, ctx.stream, a, sw_full);
            return e != cudaSuccess ? e : cudaGetLastError();
        }
    }
    const size_t smem = fixed + tree_smem_lists(rows_l, sw);
    // otherwise the register-queue builder whenever B + 1 slots fit in four registers per lane
    const bool full = sw == sw_full;
    void (*kern)(TreeArgs, int) =
        B + 1 <= 32    ? (full ? build_tree_reg_kernel<1, true> : build_tree_reg_kernel<1, false>)
        : B + 1 <= 64  ? (full ? build_tree_reg_kernel<2, true> : build_tree_reg_kernel<2, false>)
        : B + 1 <= 96  ? (full ? build_tree_reg_kernel<3, true> : build_tree_reg_kernel<3, false>)
        : B + 1 <= 128 ? (full ? build_tree_reg_kernel<4, true> : build_tree_reg_kernel<4, false>)
                       : build_tree_kernel;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    e = launch_pdl(kern, dim3(b), dim3(kTreeThreads), smem, ctx.stream, a, sw);
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t launch_tree_mask(const Ctx& ctx, int b, int B, const int32_t* node_parent, const int32_t* node_depth,
                             const int32_t* root_pos, uint8_t* mask, int32_t* pos_ids) {
    const int n = B + 1;
    const int W = (n + 31) / 32;
    const size_t smem = static_cast<size_t>(2 * n + kMaskRows * W) * 4;
    cudaError_t e = cudaFuncSetAttribute(tree_mask_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    e = launch_pdl(tree_mask_kernel, dim3(b, (n + kMaskRows - 1) / kMaskRows), dim3(256), smem, ctx.stream, n,
                   node_parent, node_depth, root_pos, mask, pos_ids);
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t launch_accept_walk(const Ctx& ctx, int b, int B, int gamma, const int32_t* node_tok,
                               const int32_t* node_parent, const int32_t* verifier_tok, int32_t* accept_len,
                               int32_t* accept_path, int32_t* next_tok) {
    const cudaError_t e = launch_pdl(accept_walk_kernel, dim3(b), dim3(32), 0, ctx.stream, B + 1, gamma, node_tok,
                                     node_parent, verifier_tok, accept_len, accept_path, next_tok);
    return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace tf
