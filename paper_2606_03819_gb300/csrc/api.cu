// C ABI of the TreeFlash drafting path (declared in include/treeflash.h): argument checks,
// workspace layout and the kernel sequence of every call. No allocation; the only global state
// is the cached driver entry point used to build TMA descriptors, a launch counter and the CUDA
// graphs of the host-buffer step (tf_draft_tree_host).
#include <math.h>
#include <string.h>

#include <algorithm>
#include <atomic>
#include <mutex>
#include <vector>

#include "common.cuh"

namespace tf {
size_t merge_smem_bytes(int n_tiles, int d, int k);

namespace {
std::atomic<unsigned long long> g_kernel_launches{0};
std::atomic<unsigned long long> g_wait_limit_ns{0};
}
void note_launch() { g_kernel_launches.fetch_add(1, std::memory_order_relaxed); }
unsigned long long wait_limit_ns() { return g_wait_limit_ns.load(std::memory_order_relaxed); }
}  // namespace tf

namespace {

using namespace tf;

constexpr size_t kAlign = 256;
constexpr size_t kMaxMergeSmem = 220 * 1024;

size_t up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

struct Dims {
    int b, d, V, I, gamma, M, K2, B, K1, R, dtype, mode, approx, n_tiles;
    int two_prev;     // TF_APPROX_SWIGLU_2PREV in TF_MODE_AR: two embeddings per row
    int k_in;         // width of the approximator input x: 2d, or 3d with two_prev
    int root_stride;  // int32 entries per sequence in root_tok: 1, or 2 with two_prev
    size_t esize;
    float inv_temp, eps;
};

struct Layout {
    size_t status, halves, chunks, X, A, hp, hres, kpart, kpart_bytes;
    size_t h_hidden, h_root, h_pos, top_ids, top_logp, child_ids, child_logp;
    size_t n_tok, n_par, n_dep, n_score, n_mask, n_pos, n_stat;
    size_t total;
};

tf_status check_dims(const tf_dims* dims, Dims* o) {
    if (!dims) return TF_ERR_INVALID_ARG;
    const tf_dims& d = *dims;
    if (d.batch < 1 || d.d < 1 || d.V < 1 || d.gamma < 1 || d.M < 1 || d.K2 < 1 || d.B < 1)
        return TF_ERR_INVALID_ARG;
    if (d.dtype != TF_BF16 && d.dtype != TF_F32) return TF_ERR_INVALID_ARG;
    if (d.mode != TF_MODE_AR && d.mode != TF_MODE_MARGINAL && d.mode != TF_MODE_MARGINAL_MARY)
        return TF_ERR_INVALID_ARG;
    if (d.mode == TF_MODE_AR && d.approx != TF_APPROX_SWIGLU && d.approx != TF_APPROX_LINEAR &&
        d.approx != TF_APPROX_SWIGLU_2PREV)
        return TF_ERR_INVALID_ARG;
    const bool two_prev = d.mode == TF_MODE_AR && d.approx == TF_APPROX_SWIGLU_2PREV;
    const bool swiglu = d.mode == TF_MODE_AR && (d.approx == TF_APPROX_SWIGLU || two_prev);
    if (!(d.temperature > 0.0f) || !isfinite(d.temperature)) return TF_ERR_INVALID_ARG;
    if (!(d.rms_eps >= 0.0f) || !isfinite(d.rms_eps)) return TF_ERR_INVALID_ARG;
    const int K1 = d.M > d.K2 ? d.M : d.K2;
    if (K1 > d.V) return TF_ERR_INVALID_ARG;
    if (swiglu && d.I < 1) return TF_ERR_INVALID_ARG;
    if (d.gamma > kMaxGamma || d.M > kMaxM || d.K2 > kMaxK || d.B > kMaxB) return TF_ERR_UNSUPPORTED;
    if (d.dtype == TF_BF16 && (d.d % 64 != 0 || (swiglu && d.I % 64 != 0)))
        return TF_ERR_UNSUPPORTED;
    const int n_tiles = (d.V + kBlockV - 1) / kBlockV;
    if (merge_smem_bytes(n_tiles, d.d, K1) > kMaxMergeSmem) return TF_ERR_UNSUPPORTED;
    // stage-2 rows per sequence: one for depth 1 and M per deeper depth; with two previous tokens
    // M for depth 2 and M^2 per depth from 3 on
    const long long M = d.M;
    const long long R = !two_prev ? 1 + M * (d.gamma - 1) : d.gamma == 1 ? 1 : 1 + M + M * M * (d.gamma - 2);
    if (static_cast<long long>(d.batch) * R > (1ll << 30) || static_cast<long long>(d.batch) * d.gamma > (1ll << 30))
        return TF_ERR_UNSUPPORTED;
    o->b = d.batch;
    o->d = d.d;
    o->V = d.V;
    o->I = swiglu ? d.I : 0;   // no SwiGLU intermediate otherwise
    o->gamma = d.gamma;
    o->M = d.M;
    o->K2 = d.K2;
    o->B = d.B;
    o->K1 = K1;
    o->R = static_cast<int>(R);
    o->dtype = d.dtype;
    o->mode = d.mode;
    o->approx = d.mode == TF_MODE_AR ? d.approx : TF_APPROX_SWIGLU;
    o->n_tiles = n_tiles;
    o->two_prev = two_prev ? 1 : 0;
    o->k_in = (two_prev ? 3 : 2) * d.d;
    o->root_stride = two_prev ? 2 : 1;
    o->esize = d.dtype == TF_BF16 ? 2 : 4;
    o->inv_temp = 1.0f / d.temperature;
    o->eps = d.rms_eps;
    return TF_OK;
}

Layout layout(const Dims& D) {
    Layout L{};
    size_t off = 0;
    auto take = [&](size_t bytes) {
        const size_t at = off;
        off += up(bytes);
        return at;
    };
    const size_t rows1 = static_cast<size_t>(D.b) * D.gamma;
    const size_t rows2 = D.mode == TF_MODE_AR ? static_cast<size_t>(D.b) * D.R : 0;
    const size_t rows = rows1 > rows2 ? rows1 : rows2;
    const size_t nn = static_cast<size_t>(D.b) * (D.B + 1);
    L.status = take(sizeof(int32_t) * (1 + kTailSems));   // the status word, then the tail-split counters
    L.halves = take(rows * D.n_tiles * kHalfBytesPerRowBlock);
    L.chunks = take(rows * D.n_tiles * kChunkBytesPerRowBlock);
    L.X = take(rows2 * D.k_in * D.esize);
    L.A = take(rows2 * D.I * D.esize);
    L.hp = take(rows2 * D.d * D.esize);
    L.hres = take(D.two_prev ? rows2 * D.d * D.esize : 0);   // residual row of each stage-2 row
    // split-K partial sums of the bf16 approximator GEMMs: [k_splits][max(2I, d) / 4][rows][4] fp32,
    // or the exchange area of their cluster path, whichever is larger
    if (D.dtype == TF_BF16) {
        const size_t partial = static_cast<size_t>(kMaxKSplits) * rows2 *
                               (2 * static_cast<size_t>(D.I) > static_cast<size_t>(D.d) ? 2 * D.I : D.d) * 4;
        const size_t xg = std::max(splitk_exchange_bytes(D.I, 2), splitk_exchange_bytes(D.d, 1));
        L.kpart_bytes = rows2 > 0 ? std::max(partial, xg) : 0;
        L.kpart = take(L.kpart_bytes);
    } else {
        L.kpart_bytes = 0;
        L.kpart = take(0);
    }
    L.h_hidden = take(rows1 * D.d * D.esize);
    L.h_root = take(static_cast<size_t>(D.b) * D.root_stride * sizeof(int32_t));
    L.h_pos = take(D.b * sizeof(int32_t));
    L.top_ids = take(rows1 * D.K1 * sizeof(int32_t));
    L.top_logp = take(rows1 * D.K1 * sizeof(float));
    L.child_ids = take(rows2 * D.K2 * sizeof(int32_t));
    L.child_logp = take(rows2 * D.K2 * sizeof(float));
    L.n_tok = take(nn * sizeof(int32_t));
    L.n_par = take(nn * sizeof(int32_t));
    L.n_dep = take(nn * sizeof(int32_t));
    L.n_score = take(nn * sizeof(float));
    L.n_mask = take(static_cast<size_t>(D.b) * (D.B + 1) * (D.B + 1));
    L.n_pos = take(nn * sizeof(int32_t));
    L.n_stat = take(D.b * sizeof(int32_t));
    L.total = off;
    return L;
}

tf_status check_ws(const Layout& L, const void* ws, size_t ws_bytes) {
    if (!ws) return TF_ERR_WORKSPACE;
    if (reinterpret_cast<uintptr_t>(ws) % kAlign != 0) return TF_ERR_WORKSPACE;
    if (ws_bytes < L.total) return TF_ERR_WORKSPACE;
    return TF_OK;
}

bool aligned16(const void* p) { return p && reinterpret_cast<uintptr_t>(p) % 16 == 0; }

template <typename P>
P* at(void* ws, size_t off) {
    return reinterpret_cast<P*>(static_cast<uint8_t*>(ws) + off);
}

tf_status make_ctx(void* ws, const Layout& L, tf_stream_t stream, Ctx* ctx) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return TF_ERR_CUDA;
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 1)
        return TF_ERR_CUDA;
    ctx->stream = reinterpret_cast<cudaStream_t>(stream);
    ctx->num_sms = sms;
    ctx->status = at<int>(ws, L.status);
    return TF_OK;
}

tf_status cuda_status(cudaError_t e) { return e == cudaSuccess ? TF_OK : TF_ERR_CUDA; }

#define TF_TRY(expr)                    \
    do {                                \
        const tf_status _s = (expr);    \
        if (_s != TF_OK) return _s;     \
    } while (0)

// ---- the pieces -----------------------------------------------------------------------------
// The LM-head partials of n_rows rows, laid out for exactly that many rows (the merge of the same
// rows reads them with the same n_rows).
Partials partials_of(const Layout& L, void* ws, int n_rows) {
    return Partials{at<float4>(ws, L.halves), at<float4>(ws, L.chunks), n_rows};
}

tf_status do_partials(const Ctx& ctx, const Dims& D, const Layout& L, void* ws, const void* lm_head, const void* x,
                      int n_rows, bool reset_status = false) {
    const Partials partials = partials_of(L, ws, n_rows);
    if (D.dtype == TF_BF16)
        return cuda_status(launch_lmhead_tc(ctx, lm_head, x, n_rows, D.d, D.V, D.inv_temp, partials, reset_status));
    return cuda_status(
        launch_lmhead_simt(ctx, D.dtype, lm_head, x, n_rows, D.d, D.V, D.inv_temp, partials, reset_status));
}

tf_status do_merge(const Ctx& ctx, const Dims& D, const Layout& L, void* ws, const void* lm_head, const void* x,
                   int n_rows, int k, int32_t* ids, float* logp) {
    return cuda_status(launch_lmhead_merge(ctx, D.dtype, partials_of(L, ws, n_rows), n_rows, D.V, D.d, k,
                                           D.inv_temp, lm_head, x, ids, logp));
}

tf_status do_ar_approx(const Ctx& ctx, const Dims& D, const Layout& L, void* ws, const tf_weights* w,
                       const void* hidden, const int32_t* root_tok, const int32_t* top_ids) {
    void* X = at<void>(ws, L.X);
    void* A = at<void>(ws, L.A);
    void* hp = at<void>(ws, L.hp);
    void* hres = at<void>(ws, L.hres);
    TF_TRY(cuda_status(launch_gather_norm(ctx, D.dtype, hidden, w->embed, w->norm_h, w->norm_e, root_tok, top_ids,
                                          D.b, D.gamma, D.M, D.K1, D.R, D.two_prev, D.d, D.V, D.eps, X,
                                          D.two_prev ? hres : nullptr)));
    const int rows = D.b * D.R;
    if (D.approx == TF_APPROX_LINEAR) {
        if (D.dtype == TF_BF16)
            return cuda_status(launch_linear_tc(ctx, X, w->w_lin, hidden, rows, D.d, D.R, D.M, D.gamma, hp,
                                                at<float>(ws, L.kpart), L.kpart_bytes));
        return cuda_status(launch_linear_simt(ctx, X, w->w_lin, hidden, rows, D.d, D.R, D.M, D.gamma, hp));
    }
    // the residual of stage-2 row r is the hidden state of its depth; with two previous tokens the
    // gather has copied it to row r of hres, which the identity map (R = M = gamma = 1) reads
    const void* res = D.two_prev ? hres : hidden;
    const int rR = D.two_prev ? 1 : D.R, rM = D.two_prev ? 1 : D.M, rG = D.two_prev ? 1 : D.gamma;
    if (D.dtype == TF_BF16)
        return cuda_status(launch_swiglu_tc(ctx, X, D.k_in, w->w_gate, w->w_up, w->w_down, res, rows, D.d, D.I, rR, rM,
                                            rG, A, hp, at<float>(ws, L.kpart), L.kpart_bytes));
    return cuda_status(launch_swiglu_simt(ctx, X, D.k_in, w->w_gate, w->w_up, w->w_down, res, rows, D.d, D.I, rR,
                                          rM, rG, A, hp));
}

tf_status check_weights(const Dims& D, const tf_weights* w, bool need_mlp) {
    if (!w || !aligned16(w->lm_head)) return TF_ERR_INVALID_ARG;
    if (!need_mlp) return TF_OK;
    if (!aligned16(w->embed) || !aligned16(w->norm_h) || !aligned16(w->norm_e)) return TF_ERR_INVALID_ARG;
    if (D.approx == TF_APPROX_LINEAR) return aligned16(w->w_lin) ? TF_OK : TF_ERR_INVALID_ARG;
    if (!aligned16(w->w_gate) || !aligned16(w->w_up) || !aligned16(w->w_down)) return TF_ERR_INVALID_ARG;
    return TF_OK;
}

struct Prepared {
    Dims D;
    Layout L;
    Ctx ctx;
};

// Host-side checks of dims and workspace (no CUDA call), then the launch context.
tf_status validate(const tf_dims* dims, void* ws, size_t ws_bytes, Prepared* p) {
    TF_TRY(check_dims(dims, &p->D));
    p->L = layout(p->D);
    return check_ws(p->L, ws, ws_bytes);
}

tf_status prepare(const tf_dims* dims, void* ws, size_t ws_bytes, tf_stream_t stream, Prepared* p) {
    TF_TRY(validate(dims, ws, ws_bytes, p));
    return make_ctx(ws, p->L, stream, &p->ctx);
}

// ---- the host-buffer step ---------------------------------------------------------------------
struct HostStep {
    const tf_dims* dims;
    const tf_weights* w;
    const void* hidden;
    const int32_t* root_tok;
    const int32_t* root_pos;
    int32_t *node_tok, *node_parent, *node_depth;
    float* node_score;
    uint8_t* mask;
    int32_t *pos_ids, *dev_status;
    void* ws;
    size_t ws_bytes;
    tf_stream_t stream;
};

// Device-visible addresses of page-locked host buffers (the same memory), or all null.
struct Mapped {
    const int32_t *root_tok, *root_pos;
    int32_t *node_tok, *node_parent, *node_depth;
    float* node_score;
    uint8_t* mask;
    int32_t *pos_ids, *dev_status;
    bool ok;
};

// The address under which the device reaches page-locked host memory `ptr`, or null.
void* device_view(const void* ptr) {
    cudaPointerAttributes a;
    if (cudaPointerGetAttributes(&a, ptr) != cudaSuccess) {
        (void)cudaGetLastError();
        return nullptr;
    }
    return a.type == cudaMemoryTypeHost ? a.devicePointer : nullptr;
}

Mapped map_host_buffers(const HostStep& h) {
    Mapped m{};
    m.root_tok = static_cast<const int32_t*>(device_view(h.root_tok));
    m.root_pos = static_cast<const int32_t*>(device_view(h.root_pos));
    m.node_tok = static_cast<int32_t*>(device_view(h.node_tok));
    m.node_parent = static_cast<int32_t*>(device_view(h.node_parent));
    m.node_depth = static_cast<int32_t*>(device_view(h.node_depth));
    m.node_score = static_cast<float*>(device_view(h.node_score));
    m.mask = static_cast<uint8_t*>(device_view(h.mask));
    m.pos_ids = static_cast<int32_t*>(device_view(h.pos_ids));
    m.dev_status = static_cast<int32_t*>(device_view(h.dev_status));
    m.ok = m.root_tok && m.root_pos && m.node_tok && m.node_parent && m.node_depth && m.node_score && m.mask &&
           m.pos_ids && m.dev_status;
    return m;
}

// Enqueues the whole host-buffer step on the stream, without synchronising: the hidden states to
// the workspace, stage 1, stage 2, the tree and its mask (dev_status with the workspace status
// word folded in by the builder, so no separate read is needed). With page-locked buffers that
// the device can address (m.ok) the kernels read root_tok / root_pos and write the outputs in
// host memory directly; otherwise those go through the workspace and copies.
tf_status enqueue_host_step(const Prepared& p, const HostStep& h, const Mapped& m) {
    const Dims& D = p.D;
    const Layout& L = p.L;
    const Ctx& ctx = p.ctx;
    cudaStream_t st = ctx.stream;
    void* ws = h.ws;
    const size_t nn = static_cast<size_t>(D.b) * (D.B + 1);
    void* d_hidden = at<void>(ws, L.h_hidden);
    TF_TRY(cuda_status(cudaMemcpyAsync(d_hidden, h.hidden, static_cast<size_t>(D.b) * D.gamma * D.d * D.esize,
                                       cudaMemcpyHostToDevice, st)));
    const int32_t* d_root = m.root_tok;
    const int32_t* d_pos = m.root_pos;
    if (!m.ok) {
        int32_t* r = at<int32_t>(ws, L.h_root);
        int32_t* q = at<int32_t>(ws, L.h_pos);
        TF_TRY(cuda_status(cudaMemcpyAsync(r, h.root_tok, static_cast<size_t>(D.b) * D.root_stride * sizeof(int32_t),
                                           cudaMemcpyHostToDevice, st)));
        TF_TRY(cuda_status(cudaMemcpyAsync(q, h.root_pos, D.b * sizeof(int32_t), cudaMemcpyHostToDevice, st)));
        d_root = r;
        d_pos = q;
    }
    int32_t* top_ids = at<int32_t>(ws, L.top_ids);
    float* top_logp = at<float>(ws, L.top_logp);
    int32_t* child_ids = at<int32_t>(ws, L.child_ids);
    float* child_logp = at<float>(ws, L.child_logp);
    TF_TRY(tf_stage1_marginals(h.dims, h.w, d_hidden, top_ids, top_logp, ws, h.ws_bytes, h.stream));
    if (D.mode == TF_MODE_AR)
        TF_TRY(tf_stage2_ar_approx(h.dims, h.w, d_hidden, d_root, top_ids, child_ids, child_logp, ws, h.ws_bytes,
                                   h.stream));
    int32_t* o_tok = m.ok ? m.node_tok : at<int32_t>(ws, L.n_tok);
    int32_t* o_par = m.ok ? m.node_parent : at<int32_t>(ws, L.n_par);
    int32_t* o_dep = m.ok ? m.node_depth : at<int32_t>(ws, L.n_dep);
    float* o_score = m.ok ? m.node_score : at<float>(ws, L.n_score);
    uint8_t* o_mask = m.ok ? m.mask : at<uint8_t>(ws, L.n_mask);
    int32_t* o_pos = m.ok ? m.pos_ids : at<int32_t>(ws, L.n_pos);
    int32_t* o_stat = m.ok ? m.dev_status : at<int32_t>(ws, L.n_stat);
    const bool ar = D.mode == TF_MODE_AR;
    const bool fused = D.B + 1 <= kFusedMaskMaxNodes;   // the builder CTA writes the mask of its tree
    TF_TRY(cuda_status(launch_build_tree(ctx, D.b, D.gamma, D.M, D.K1, D.K2, D.B, D.V, D.mode, D.R, D.two_prev, d_root,
                                         top_ids, top_logp, ar ? child_ids : nullptr, ar ? child_logp : nullptr, o_tok,
                                         o_par, o_dep, o_score, o_stat, fused ? d_pos : nullptr, fused ? o_mask : nullptr,
                                         fused ? o_pos : nullptr, ctx.status)));
    if (!fused) TF_TRY(cuda_status(launch_tree_mask(ctx, D.b, D.B, o_par, o_dep, d_pos, o_mask, o_pos)));
    if (m.ok) return TF_OK;
    TF_TRY(cuda_status(cudaMemcpyAsync(h.node_tok, o_tok, nn * 4, cudaMemcpyDeviceToHost, st)));
    TF_TRY(cuda_status(cudaMemcpyAsync(h.node_parent, o_par, nn * 4, cudaMemcpyDeviceToHost, st)));
    TF_TRY(cuda_status(cudaMemcpyAsync(h.node_depth, o_dep, nn * 4, cudaMemcpyDeviceToHost, st)));
    TF_TRY(cuda_status(cudaMemcpyAsync(h.node_score, o_score, nn * 4, cudaMemcpyDeviceToHost, st)));
    TF_TRY(cuda_status(cudaMemcpyAsync(h.mask, o_mask, nn * (D.B + 1), cudaMemcpyDeviceToHost, st)));
    TF_TRY(cuda_status(cudaMemcpyAsync(h.pos_ids, o_pos, nn * 4, cudaMemcpyDeviceToHost, st)));
    return cuda_status(cudaMemcpyAsync(h.dev_status, o_stat, D.b * 4, cudaMemcpyDeviceToHost, st));
}

// The host-buffer step as a CUDA graph, captured on the first call with a given set of arguments
// and replayed afterwards: one graph launch in place of three copies, eight to nine kernel launches
// and seven copies, and the next step's first kernel no longer waits for the host to issue it.
// Only for a created stream (the legacy default stream cannot be captured) and page-locked host
// buffers (copies from pageable memory cannot be captured); otherwise, or when the capture or the
// instantiation fails, the step runs as plain launches. The key holds everything the captured
// kernels and copies read at capture time: dims, weight, buffer and workspace pointers, the device
// and the wait limit of the tensor-core kernels. At most kMaxHostGraphs are kept (oldest evicted).
struct HostGraph {
    std::vector<uint64_t> key;
    cudaGraphExec_t exec;       // nullptr: this step could not be captured, run it as plain launches
    unsigned long long kernels; // kernel launches in the graph (for the library's launch counter)
};
std::mutex g_host_graph_mu;
std::vector<HostGraph> g_host_graphs;
constexpr size_t kMaxHostGraphs = 8;

uint32_t float_bits(float f) {
    uint32_t u;
    memcpy(&u, &f, sizeof(u));
    return u;
}

bool page_locked(const void* ptr) {
    cudaPointerAttributes a;
    if (cudaPointerGetAttributes(&a, ptr) != cudaSuccess) {
        (void)cudaGetLastError();
        return false;
    }
    return a.type == cudaMemoryTypeHost;
}

tf_status launch_host_graph(const Prepared& p, const HostStep& h, const Mapped& m, bool* replayed) {
    *replayed = false;
    cudaStream_t st = p.ctx.stream;
    if (st == nullptr || st == cudaStreamLegacy || st == cudaStreamPerThread) return TF_OK;
    cudaStreamCaptureStatus cs;
    if (cudaStreamIsCapturing(st, &cs) != cudaSuccess) {
        (void)cudaGetLastError();
        return TF_OK;
    }
    if (cs != cudaStreamCaptureStatusNone) return TF_OK;
    const void* host_ptrs[] = {h.hidden, h.root_tok, h.root_pos, h.node_tok, h.node_parent, h.node_depth,
                               h.node_score, h.mask, h.pos_ids, h.dev_status};
    for (const void* q : host_ptrs)
        if (!page_locked(q)) return TF_OK;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return TF_ERR_CUDA;
    const tf_dims& d = *h.dims;
    std::vector<uint64_t> key = {
        static_cast<uint64_t>(d.batch), static_cast<uint64_t>(d.d), static_cast<uint64_t>(d.V), static_cast<uint64_t>(d.I),
        static_cast<uint64_t>(d.gamma), static_cast<uint64_t>(d.M), static_cast<uint64_t>(d.K2), static_cast<uint64_t>(d.B),
        static_cast<uint64_t>(float_bits(d.temperature)), static_cast<uint64_t>(float_bits(d.rms_eps)),
        static_cast<uint64_t>(d.dtype), static_cast<uint64_t>(d.mode), static_cast<uint64_t>(d.approx),
        static_cast<uint64_t>(dev), wait_limit_ns(), reinterpret_cast<uint64_t>(h.ws), static_cast<uint64_t>(h.ws_bytes)};
    const void* w_ptrs[] = {h.w->lm_head, h.w->embed, h.w->norm_h, h.w->norm_e, h.w->w_gate, h.w->w_up, h.w->w_down,
                            h.w->w_lin};
    for (const void* q : w_ptrs) key.push_back(reinterpret_cast<uint64_t>(q));
    for (const void* q : host_ptrs) key.push_back(reinterpret_cast<uint64_t>(q));

    std::lock_guard<std::mutex> lock(g_host_graph_mu);
    HostGraph* hit = nullptr;
    for (auto& g : g_host_graphs)
        if (g.key == key) hit = &g;
    if (!hit) {
        if (cudaStreamBeginCapture(st, cudaStreamCaptureModeThreadLocal) != cudaSuccess) {
            (void)cudaGetLastError();
            return TF_OK;
        }
        // captured launches run only with the graph: they are counted at each replay instead
        const unsigned long long c0 = tf::g_kernel_launches.load(std::memory_order_relaxed);
        const tf_status es = enqueue_host_step(p, h, m);
        const unsigned long long kernels = tf::g_kernel_launches.load(std::memory_order_relaxed) - c0;
        tf::g_kernel_launches.fetch_sub(kernels, std::memory_order_relaxed);
        cudaGraph_t graph = nullptr;
        const cudaError_t ce = cudaStreamEndCapture(st, &graph);
        cudaGraphExec_t exec = nullptr;
        if (es == TF_OK && ce == cudaSuccess && graph &&
            cudaGraphInstantiate(&exec, graph, 0) != cudaSuccess)
            exec = nullptr;
        if (graph) cudaGraphDestroy(graph);
        (void)cudaGetLastError();
        if (es != TF_OK && es != TF_ERR_CUDA) return es;   // an argument error: nothing to cache
        if (g_host_graphs.size() >= kMaxHostGraphs) {
            if (g_host_graphs.front().exec) cudaGraphExecDestroy(g_host_graphs.front().exec);
            g_host_graphs.erase(g_host_graphs.begin());
        }
        g_host_graphs.push_back(HostGraph{key, exec, kernels});
        hit = &g_host_graphs.back();
    }
    if (!hit->exec) return TF_OK;
    if (cudaGraphLaunch(hit->exec, st) != cudaSuccess) return TF_ERR_CUDA;
    tf::g_kernel_launches.fetch_add(hit->kernels, std::memory_order_relaxed);
    *replayed = true;
    return TF_OK;
}

}  // namespace

extern "C" {

const char* tf_status_string(tf_status s) {
    switch (s) {
        case TF_OK: return "ok";
        case TF_ERR_INVALID_ARG: return "invalid argument";
        case TF_ERR_UNSUPPORTED: return "unsupported dimensions";
        case TF_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
        case TF_ERR_CUDA: return "CUDA error";
        case TF_ERR_DEVICE_STATUS: return "device reported a condition (TF_DEV_* flags)";
        case TF_ERR_TIMEOUT: return "a bounded device wait gave up";
    }
    return "unknown status";
}

int32_t tf_version(void) { return 100; }

uint64_t tf_kernel_launches(void) { return tf::g_kernel_launches.load(std::memory_order_relaxed); }

tf_status tf_set_wait_limit_ns(uint64_t ns) {
    if (ns > 60ull * 1000000000ull) return TF_ERR_INVALID_ARG;
    tf::g_wait_limit_ns.store(ns, std::memory_order_relaxed);
    return TF_OK;
}

tf_status tf_workspace_size(const tf_dims* dims, size_t* bytes) {
    if (!bytes) return TF_ERR_INVALID_ARG;
    Dims D;
    TF_TRY(check_dims(dims, &D));
    *bytes = layout(D).total;
    return TF_OK;
}

tf_status tf_status_reset(void* ws, size_t ws_bytes, tf_stream_t stream) {
    if (!ws || ws_bytes < sizeof(int32_t) || reinterpret_cast<uintptr_t>(ws) % kAlign) return TF_ERR_WORKSPACE;
    return cuda_status(cudaMemsetAsync(ws, 0, sizeof(int32_t), reinterpret_cast<cudaStream_t>(stream)));
}

tf_status tf_status_read(const void* ws, size_t ws_bytes, int32_t* flags, tf_stream_t stream) {
    if (!flags) return TF_ERR_INVALID_ARG;
    if (!ws || ws_bytes < sizeof(int32_t) || reinterpret_cast<uintptr_t>(ws) % kAlign) return TF_ERR_WORKSPACE;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    int32_t v = 0;
    if (cudaMemcpyAsync(&v, ws, sizeof(int32_t), cudaMemcpyDeviceToHost, st) != cudaSuccess) return TF_ERR_CUDA;
    if (cudaStreamSynchronize(st) != cudaSuccess) return TF_ERR_CUDA;
    *flags = v;
    if (v & TF_DEV_TIMEOUT) return TF_ERR_TIMEOUT;
    if (v & ~TF_DEV_RECOMPUTED) return TF_ERR_DEVICE_STATUS;
    return TF_OK;
}

tf_status tf_lmhead_partials(const tf_dims* dims, const void* lm_head, const void* x, int32_t n_rows, void* ws,
                             size_t ws_bytes, tf_stream_t stream) {
    Prepared p;
    TF_TRY(prepare(dims, ws, ws_bytes, stream, &p));
    const long long max_rows = std::max(static_cast<long long>(p.D.b) * p.D.gamma,
                                        p.D.mode == TF_MODE_AR ? static_cast<long long>(p.D.b) * p.D.R : 0ll);
    if (!aligned16(lm_head) || !aligned16(x) || n_rows < 0 || n_rows > max_rows) return TF_ERR_INVALID_ARG;
    return do_partials(p.ctx, p.D, p.L, ws, lm_head, x, n_rows);
}

tf_status tf_lmhead_merge(const tf_dims* dims, const void* lm_head, const void* x, int32_t n_rows, int32_t k,
                          int32_t* out_ids, float* out_logp, void* ws, size_t ws_bytes, tf_stream_t stream) {
    Prepared p;
    TF_TRY(prepare(dims, ws, ws_bytes, stream, &p));
    const long long max_rows = std::max(static_cast<long long>(p.D.b) * p.D.gamma,
                                        p.D.mode == TF_MODE_AR ? static_cast<long long>(p.D.b) * p.D.R : 0ll);
    if (!lm_head || !x || !out_ids || !out_logp || n_rows < 0 || n_rows > max_rows) return TF_ERR_INVALID_ARG;
    if (k < 1 || k > kMaxK || k > p.D.V) return TF_ERR_INVALID_ARG;
    return do_merge(p.ctx, p.D, p.L, ws, lm_head, x, n_rows, k, out_ids, out_logp);
}

tf_status tf_stage1_marginals(const tf_dims* dims, const tf_weights* w, const void* hidden, int32_t* top_ids,
                              float* top_logp, void* ws, size_t ws_bytes, tf_stream_t stream) {
    Prepared p;
    TF_TRY(validate(dims, ws, ws_bytes, &p));
    TF_TRY(check_weights(p.D, w, false));
    if (!aligned16(hidden) || !top_ids || !top_logp) return TF_ERR_INVALID_ARG;
    TF_TRY(make_ctx(ws, p.L, stream, &p.ctx));
    const int rows = p.D.b * p.D.gamma;
    TF_TRY(do_partials(p.ctx, p.D, p.L, ws, w->lm_head, hidden, rows, /*reset_status=*/true));
    return do_merge(p.ctx, p.D, p.L, ws, w->lm_head, hidden, rows, p.D.K1, top_ids, top_logp);
}

tf_status tf_ar_approx(const tf_dims* dims, const tf_weights* w, const void* hidden, const int32_t* root_tok,
                       const int32_t* top_ids, void* h_prime, void* ws, size_t ws_bytes, tf_stream_t stream) {
    Prepared p;
    TF_TRY(validate(dims, ws, ws_bytes, &p));
    if (p.D.mode != TF_MODE_AR) return TF_ERR_INVALID_ARG;
    TF_TRY(check_weights(p.D, w, true));
    if (!aligned16(hidden) || !root_tok || !top_ids) return TF_ERR_INVALID_ARG;
    TF_TRY(make_ctx(ws, p.L, stream, &p.ctx));
    TF_TRY(do_ar_approx(p.ctx, p.D, p.L, ws, w, hidden, root_tok, top_ids));
    if (h_prime) {
        const size_t bytes = static_cast<size_t>(p.D.b) * p.D.R * p.D.d * p.D.esize;
        TF_TRY(cuda_status(cudaMemcpyAsync(h_prime, at<void>(ws, p.L.hp), bytes, cudaMemcpyDeviceToDevice,
                                           p.ctx.stream)));
    }
    return TF_OK;
}

tf_status tf_stage2_ar_approx(const tf_dims* dims, const tf_weights* w, const void* hidden, const int32_t* root_tok,
                              const int32_t* top_ids, int32_t* child_ids, float* child_logp, void* ws,
                              size_t ws_bytes, tf_stream_t stream) {
    Prepared p;
    TF_TRY(validate(dims, ws, ws_bytes, &p));
    if (p.D.mode != TF_MODE_AR) return TF_ERR_INVALID_ARG;
    TF_TRY(check_weights(p.D, w, true));
    if (!aligned16(hidden) || !root_tok || !top_ids || !child_ids || !child_logp) return TF_ERR_INVALID_ARG;
    TF_TRY(make_ctx(ws, p.L, stream, &p.ctx));
    TF_TRY(do_ar_approx(p.ctx, p.D, p.L, ws, w, hidden, root_tok, top_ids));
    const int rows = p.D.b * p.D.R;
    const void* hp = at<void>(ws, p.L.hp);
    TF_TRY(do_partials(p.ctx, p.D, p.L, ws, w->lm_head, hp, rows));
    return do_merge(p.ctx, p.D, p.L, ws, w->lm_head, hp, rows, p.D.K2, child_ids, child_logp);
}

tf_status tf_build_tree(const tf_dims* dims, const int32_t* root_tok, const int32_t* top_ids, const float* top_logp,
                        const int32_t* child_ids, const float* child_logp, int32_t* node_tok, int32_t* node_parent,
                        int32_t* node_depth, float* node_score, int32_t* dev_status, tf_stream_t stream) {
    Dims D;
    TF_TRY(check_dims(dims, &D));
    if (!root_tok || !top_ids || !top_logp || !node_tok || !node_parent || !node_depth || !node_score || !dev_status)
        return TF_ERR_INVALID_ARG;
    if (D.mode == TF_MODE_AR && (!child_ids || !child_logp)) return TF_ERR_INVALID_ARG;
    Ctx ctx{reinterpret_cast<cudaStream_t>(stream), 0, nullptr};
    return cuda_status(launch_build_tree(ctx, D.b, D.gamma, D.M, D.K1, D.K2, D.B, D.V, D.mode, D.R, D.two_prev,
                                         root_tok, top_ids, top_logp, child_ids, child_logp, node_tok, node_parent,
                                         node_depth, node_score, dev_status));
}

tf_status tf_tree_mask(const tf_dims* dims, const int32_t* node_parent, const int32_t* node_depth,
                       const int32_t* root_pos, uint8_t* mask, int32_t* pos_ids, tf_stream_t stream) {
    Dims D;
    TF_TRY(check_dims(dims, &D));
    if (!node_parent || !node_depth || !root_pos || !mask || !pos_ids) return TF_ERR_INVALID_ARG;
    Ctx ctx{reinterpret_cast<cudaStream_t>(stream), 0, nullptr};
    return cuda_status(launch_tree_mask(ctx, D.b, D.B, node_parent, node_depth, root_pos, mask, pos_ids));
}

tf_status tf_build_tree_mask(const tf_dims* dims, const int32_t* root_tok, const int32_t* root_pos,
                             const int32_t* top_ids, const float* top_logp, const int32_t* child_ids,
                             const float* child_logp, int32_t* node_tok, int32_t* node_parent, int32_t* node_depth,
                             float* node_score, uint8_t* mask, int32_t* pos_ids, int32_t* dev_status,
                             tf_stream_t stream) {
    Dims D;
    TF_TRY(check_dims(dims, &D));
    if (!root_tok || !root_pos || !top_ids || !top_logp || !node_tok || !node_parent || !node_depth || !node_score ||
        !mask || !pos_ids || !dev_status)
        return TF_ERR_INVALID_ARG;
    if (D.mode == TF_MODE_AR && (!child_ids || !child_logp)) return TF_ERR_INVALID_ARG;
    Ctx ctx{reinterpret_cast<cudaStream_t>(stream), 0, nullptr};
    const bool fused = D.B + 1 <= kFusedMaskMaxNodes;   // the builder CTA writes the mask of its tree
    TF_TRY(cuda_status(launch_build_tree(ctx, D.b, D.gamma, D.M, D.K1, D.K2, D.B, D.V, D.mode, D.R, D.two_prev, root_tok,
                                         top_ids, top_logp, child_ids, child_logp, node_tok, node_parent, node_depth,
                                         node_score, dev_status, fused ? root_pos : nullptr,
                                         fused ? mask : nullptr, fused ? pos_ids : nullptr)));
    if (fused) return TF_OK;
    return cuda_status(launch_tree_mask(ctx, D.b, D.B, node_parent, node_depth, root_pos, mask, pos_ids));
}

tf_status tf_accept_walk(const tf_dims* dims, const int32_t* node_tok, const int32_t* node_parent,
                         const int32_t* verifier_tok, int32_t* accept_len, int32_t* accept_path, int32_t* next_tok,
                         tf_stream_t stream) {
    Dims D;
    TF_TRY(check_dims(dims, &D));
    if (!node_tok || !node_parent || !verifier_tok || !accept_len || !accept_path || !next_tok)
        return TF_ERR_INVALID_ARG;
    Ctx ctx{reinterpret_cast<cudaStream_t>(stream), 0, nullptr};
    return cuda_status(launch_accept_walk(ctx, D.b, D.B, D.gamma, node_tok, node_parent, verifier_tok, accept_len,
                                          accept_path, next_tok));
}

tf_status tf_workspace_h_prime(const tf_dims* dims, void* ws, size_t ws_bytes, void** h_prime) {
    if (!h_prime) return TF_ERR_INVALID_ARG;
    Dims D;
    TF_TRY(check_dims(dims, &D));
    if (D.mode != TF_MODE_AR) return TF_ERR_INVALID_ARG;
    const Layout L = layout(D);
    TF_TRY(check_ws(L, ws, ws_bytes));
    *h_prime = at<void>(ws, L.hp);
    return TF_OK;
}

tf_status tf_workspace_view(const tf_dims* dims, void* ws, size_t ws_bytes, int32_t view, void** ptr,
                            size_t* bytes) {
    if (!ptr || !bytes) return TF_ERR_INVALID_ARG;
    Dims D;
    TF_TRY(check_dims(dims, &D));
    const Layout L = layout(D);
    TF_TRY(check_ws(L, ws, ws_bytes));
    const size_t rows2 = static_cast<size_t>(D.b) * D.R;
    const size_t rows1 = static_cast<size_t>(D.b) * D.gamma;
    const size_t rows_lm = D.mode == TF_MODE_AR && rows2 > rows1 ? rows2 : rows1;
    switch (view) {
        case TF_VIEW_HALVES:
            *ptr = at<void>(ws, L.halves);
            *bytes = rows_lm * D.n_tiles * kHalfBytesPerRowBlock;
            return TF_OK;
        case TF_VIEW_CHUNKS:
            *ptr = at<void>(ws, L.chunks);
            *bytes = rows_lm * D.n_tiles * kChunkBytesPerRowBlock;
            return TF_OK;
    }
    if (D.mode != TF_MODE_AR) return TF_ERR_INVALID_ARG;
    switch (view) {
        case TF_VIEW_X: *ptr = at<void>(ws, L.X); *bytes = rows2 * D.k_in * D.esize; return TF_OK;
        case TF_VIEW_A: *ptr = at<void>(ws, L.A); *bytes = rows2 * D.I * D.esize; return TF_OK;
        case TF_VIEW_H_PRIME: *ptr = at<void>(ws, L.hp); *bytes = rows2 * D.d * D.esize; return TF_OK;
    }
    return TF_ERR_INVALID_ARG;
}

tf_status tf_draft_tree_host(const tf_dims* dims, const tf_weights* w, const void* hidden, const int32_t* root_tok,
                             const int32_t* root_pos, int32_t* node_tok, int32_t* node_parent, int32_t* node_depth,
                             float* node_score, uint8_t* mask, int32_t* pos_ids, int32_t* dev_status, void* ws,
                             size_t ws_bytes, tf_stream_t stream) {
    Prepared p;
    TF_TRY(prepare(dims, ws, ws_bytes, stream, &p));
    if (!hidden || !root_tok || !root_pos || !node_tok || !node_parent || !node_depth || !node_score || !mask ||
        !pos_ids || !dev_status)
        return TF_ERR_INVALID_ARG;
    const HostStep h{dims, w, hidden, root_tok, root_pos, node_tok, node_parent, node_depth, node_score, mask, pos_ids,
                     dev_status, ws, ws_bytes, stream};
    cudaStream_t st = p.ctx.stream;
    const Mapped m = map_host_buffers(h);
    bool replayed = false;
    TF_TRY(launch_host_graph(p, h, m, &replayed));
    if (!replayed) TF_TRY(enqueue_host_step(p, h, m));
    if (cudaStreamSynchronize(st) != cudaSuccess) return TF_ERR_CUDA;
    // every dev_status entry carries the workspace word in bits 16 and up (folded by the builder)
    const int32_t flags = dev_status[0] >> 16;
    for (int s = 0; s < p.D.b; ++s) dev_status[s] &= 0xffff;
    if (flags & TF_DEV_TIMEOUT) return TF_ERR_TIMEOUT;
    if (flags & ~TF_DEV_RECOMPUTED) return TF_ERR_DEVICE_STATUS;
    return TF_OK;
}

}  // extern "C"
