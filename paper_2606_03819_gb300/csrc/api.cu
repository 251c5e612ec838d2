// C ABI of the TreeFlash drafting path (declared in include/treeflash.h): argument checks,
// workspace layout and the kernel sequence of every call. No allocation; the only global state
// is the cached driver entry point used to build TMA descriptors and a launch counter.
#include <math.h>
#include <string.h>

#include <algorithm>
#include <atomic>

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
    const Dims& D = p.D;
    const Layout& L = p.L;
    cudaStream_t st = p.ctx.stream;
    const size_t nn = static_cast<size_t>(D.b) * (D.B + 1);
    void* d_hidden = at<void>(ws, L.h_hidden);
    int32_t* d_root = at<int32_t>(ws, L.h_root);
    int32_t* d_pos = at<int32_t>(ws, L.h_pos);
    TF_TRY(cuda_status(cudaMemcpyAsync(d_hidden, hidden, static_cast<size_t>(D.b) * D.gamma * D.d * D.esize,
                                       cudaMemcpyHostToDevice, st)));
    TF_TRY(cuda_status(cudaMemcpyAsync(d_root, root_tok, static_cast<size_t>(D.b) * D.root_stride * sizeof(int32_t),
                                       cudaMemcpyHostToDevice, st)));
    TF_TRY(cuda_status(cudaMemcpyAsync(d_pos, root_pos, D.b * sizeof(int32_t), cudaMemcpyHostToDevice, st)));
    int32_t* top_ids = at<int32_t>(ws, L.top_ids);
    float* top_logp = at<float>(ws, L.top_logp);
    int32_t* child_ids = at<int32_t>(ws, L.child_ids);
    float* child_logp = at<float>(ws, L.child_logp);
    TF_TRY(tf_stage1_marginals(dims, w, d_hidden, top_ids, top_logp, ws, ws_bytes, stream));
    if (D.mode == TF_MODE_AR)
        TF_TRY(tf_stage2_ar_approx(dims, w, d_hidden, d_root, top_ids, child_ids, child_logp, ws, ws_bytes, stream));
    int32_t* d_tok = at<int32_t>(ws, L.n_tok);
    int32_t* d_par = at<int32_t>(ws, L.n_par);
    int32_t* d_dep = at<int32_t>(ws, L.n_dep);
    float* d_score = at<float>(ws, L.n_score);
    uint8_t* d_mask = at<uint8_t>(ws, L.n_mask);
    int32_t* d_posid = at<int32_t>(ws, L.n_pos);
    int32_t* d_stat = at<int32_t>(ws, L.n_stat);
    TF_TRY(tf_build_tree_mask(dims, d_root, d_pos, top_ids, top_logp, D.mode == TF_MODE_AR ? child_ids : nullptr,
                              D.mode == TF_MODE_AR ? child_logp : nullptr, d_tok, d_par, d_dep, d_score, d_mask,
                              d_posid, d_stat, stream));
    TF_TRY(cuda_status(cudaMemcpyAsync(node_tok, d_tok, nn * 4, cudaMemcpyDeviceToHost, st)));
    TF_TRY(cuda_status(cudaMemcpyAsync(node_parent, d_par, nn * 4, cudaMemcpyDeviceToHost, st)));
    TF_TRY(cuda_status(cudaMemcpyAsync(node_depth, d_dep, nn * 4, cudaMemcpyDeviceToHost, st)));
    TF_TRY(cuda_status(cudaMemcpyAsync(node_score, d_score, nn * 4, cudaMemcpyDeviceToHost, st)));
    TF_TRY(cuda_status(cudaMemcpyAsync(mask, d_mask, nn * (D.B + 1), cudaMemcpyDeviceToHost, st)));
    TF_TRY(cuda_status(cudaMemcpyAsync(pos_ids, d_posid, nn * 4, cudaMemcpyDeviceToHost, st)));
    TF_TRY(cuda_status(cudaMemcpyAsync(dev_status, d_stat, D.b * 4, cudaMemcpyDeviceToHost, st)));
    int32_t flags = 0;
    const tf_status rs = tf_status_read(ws, ws_bytes, &flags, stream);  // synchronises the stream
    if (rs == TF_ERR_CUDA) return rs;
    for (int s = 0; s < D.b; ++s) dev_status[s] |= flags;
    return rs;
}

}  // extern "C"
