// Tensor-core (tcgen05 + TMA) GEMM kernels of the bf16 path.
//
//   D[r, n] = sum_k X[r, k] * W[n, k]          X: activations [rows, K], W: weights [N, K]
//
// X rows sit in the 128 TMEM lanes (M = 128 per tile), weight rows in the MMA N dimension, so
// every epilogue thread owns one activation row and walks its logits / outputs serially.
// Three fused epilogues:
//   LMHEAD  the LM-head pass of Algorithm 1 (stage 1 and stage 2): for each (row, block of 256
//           vocabulary entries) it keeps per half block the max, the sum of exp(z - max) and the
//           best (z, id), and per 32-wide chunk the three largest z with the ids of the first
//           two. Logits never leave the SM.
//   GATEUP  SwiGLU of Eq. 1, first half: A = SiLU(X W_gate^T) * (X W_up^T), bf16 out.
//   DOWN    SwiGLU of Eq. 1, second half plus the residual: h' = h + A W_down^T, bf16 out; the
//           same epilogue serves the linear approximator of the ablations, h' = h + x W_lin^T.
//
// Warp roles (576 threads, one CTA per SM, persistent over work units):
//   warp 0      TMA producer: one elected lane streams X and W tiles into a ring of stages.
//   warp 1      TMEM allocator and MMA issuer (one lane issues tcgen05.mma and commits).
//   warps 2..17 epilogue, two groups of eight; group g drains accumulator slot g (TMEM columns
//               [256 g, 256 g + 256)); warp w may only touch TMEM lanes 32 (w % 4) .. + 31, and
//               the two warps of a group on the same lanes split the columns in halves.
// A work unit is (N tile, group of MT M-tiles). With MT = 2 both slots hold one unit (M-tile j
// in slot j); with MT = 1 consecutive units alternate slots so the epilogue of one overlaps the
// MMAs of the next. With clusters of CL = 2 CTAs (the LM head over more than 128 rows) the two
// CTAs are a tcgen05 CTA pair: units are dealt to clusters, CTA r of a cluster stages M-tile r of
// the unit's pair of M-tiles and weight rows [128 r, 128 r + 128) of the unit's 256-row weight
// tile, and the even CTA issues one cta_group::2 MMA (M = 256, N = 256) per K slice that reads
// both CTAs' shared memory and writes each CTA's 128 rows into its own TMEM. W is read once, each
// CTA stages 32 KB per stage instead of 48 KB, and each keeps one TMEM slot per unit, so its
// epilogue overlaps the next unit's MMAs. Every wait is bounded: after a time limit the kernel
// raises TF_DEV_TIMEOUT, drains its in-flight copies and MMAs, frees TMEM and returns.
#include <cuda.h>
#include <math.h>

#include "common.cuh"
#include "tc_ptx.cuh"

namespace tf {
namespace {

constexpr int kBK = 64;       // K elements per stage: one 128-byte swizzle row of bf16
constexpr int kBM = 128;      // activation rows per M-tile (TMEM lanes)
constexpr int kEpiWarps = 16;  // two groups (one per TMEM slot) of eight warps
constexpr int kThreads = 64 + 32 * kEpiWarps;
constexpr uint64_t kWaitLimitNs = 2000000000ull;

// EPI_CGATEUP / EPI_CDOWN: the GATEUP / DOWN results from split-K over the CTAs of a cluster, the
// partial sums added in shared memory across the cluster instead of through global memory.
enum { EPI_LMHEAD = 0, EPI_GATEUP = 1, EPI_DOWN = 2, EPI_PARTIAL = 3, EPI_CGATEUP = 4, EPI_CDOWN = 5 };

struct EpiParams {
    Partials partials;           // LMHEAD: per (row, vocabulary block) summaries
    int V;
    float inv_temp;
    __nv_bfloat16* out;          // GATEUP: A [n_rows, ld_out]; DOWN: h' [n_rows, ld_out]
    int ld_out;
    const __nv_bfloat16* hidden; // DOWN: residual rows, [b * gamma, ld_out]
    int R, M, gamma;
    float* partial;              // PARTIAL: fp32 sums [k_splits][n_cols / 4][n_rows][4] (float4-major),
    int n_cols;                  //          accumulator nb of N tile nt at columns nb * n_total + nt * BN
    int n_total;                 // N of the whole GEMM (n_ntiles * BN)
    int reset_status;            // LMHEAD: zero *status first (the first kernel of a stage-1 call)
    unsigned long long wait_ns;  // limit of every wait for progress (0: kWaitLimitNs); the waits
                                 // that drain in-flight copies and MMAs always take kWaitLimitNs
    // GATEUP / DOWN with one CTA per SM: units n_full.. (the last, partial round) run as
    // tail_split K-chunks each (0: none). A chunk writes its fp32 partial sums to `partial`, laid
    // out [tail unit][chunk][M-tile][col / 4][128 rows][4]; the chunk that finishes last (counted
    // in sem[tail unit * MT + M-tile], zero between calls) adds them in chunk order and applies
    // the epilogue.
    int n_full, tail_split;
    int* sem;
};

// Work unit u -> (N tile, M-tile group, K split); consecutive units share the N tile and K split
// (the same weight tile) and differ in the M-tile group, so batched rows reuse it from L2.
struct Unit {
    int nt, mg, kx;
};
__device__ __forceinline__ Unit decode_unit(int u, int n_mgroups, int k_splits) {
    Unit w;
    w.mg = u % n_mgroups;
    const int rest = u / n_mgroups;
    w.kx = rest % k_splits;
    w.nt = rest / k_splits;
    return w;
}

// PAIR: a CTA of a cta_group::2 pair, which stages half of the weight tile (BN / 2 rows).
template <int MT, int NB, int BN, int STAGES, bool PAIR = false>
struct TileCfg {
    static constexpr int kABytes = kBM * kBK * 2;
    static constexpr int kBBytes = BN * kBK * 2;                    // the whole weight tile of a stage
    static constexpr int kBBytesCta = PAIR ? kBBytes / 2 : kBBytes;  // the part this CTA stages
    static constexpr int kStageBytes = MT * kABytes + NB * kBBytesCta;
    static constexpr int kBarrierBytes = 256;
    static constexpr int kSmemBytes = STAGES * kStageBytes + kBarrierBytes + 1024;
    static_assert(NB * BN <= 256, "one accumulator slot is 256 TMEM columns");
    static_assert(BN % 64 == 0 && BN >= 64 && BN <= 256, "N tile (two epilogue warps split it in 32-column steps)");
    static_assert(kStageBytes % 1024 == 0, "stages must stay 1024-byte aligned for 128B swizzle");
};

__device__ __forceinline__ float silu_f(float g) { return g / (1.0f + __expf(-g)); }

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&v);
}

// Summary of one 32-column chunk of one row: logits of vocabulary ids v0 .. v0+31. The three
// largest values, the chunk-local offsets of the first two (the smaller id first among equals)
// and the sum of exp(z - max) come from one fixed tree over the 32 registers: the same
// instructions for every lane whatever the data (a per-lane sorted insertion would diverge across
// the warp's 32 rows). Each node carries its subtree's top three and its sum of exp(z - node
// max), so a logit is dead once its leaf is formed; the tree is expanded depth first to keep
// few nodes live.
struct ChunkNode {
    float a1, a2, a3, s;  // a1 >= a2 >= a3; s = sum over the subtree of exp(z - a1)
    int i1, i2;           // chunk-local offsets of a1, a2
};
__device__ __forceinline__ float chunk_logit(uint32_t r, int v, int V, float inv_temp) {
    return v < V ? __uint_as_float(r) * inv_temp : -INFINITY;
}
// p covers smaller ids than q, so on equal values p's entry ranks first.
__device__ __forceinline__ ChunkNode chunk_merge(const ChunkNode& p, const ChunkNode& q) {
    const bool pw = p.a1 >= q.a1;
    const ChunkNode& w = pw ? p : q;
    const ChunkNode& l = pw ? q : p;
    // the winner's second against the loser's first; p's ids rank first on equal values
    const bool sw = pw ? (w.a2 >= l.a1) : (w.a2 > l.a1);
    ChunkNode n;
    n.a1 = w.a1;
    n.i1 = w.i1;
    n.a2 = sw ? w.a2 : l.a1;
    n.i2 = sw ? w.i2 : l.i1;
    n.a3 = sw ? fmaxf(w.a3, l.a1) : fmaxf(w.a2, l.a2);
    n.s = w.s + (l.a1 > -INFINITY ? l.s * __expf(l.a1 - w.a1) : 0.0f);
    return n;
}
template <int OFF, int N>
__device__ __forceinline__ ChunkNode chunk_tree(const uint32_t (&r)[32], int v0, int V, float inv_temp) {
    if constexpr (N == 2) {
        const float x = chunk_logit(r[OFF], v0 + OFF, V, inv_temp);
        const float y = chunk_logit(r[OFF + 1], v0 + OFF + 1, V, inv_temp);
        const bool ge = x >= y;
        ChunkNode n;
        n.a1 = ge ? x : y;
        n.a2 = ge ? y : x;
        n.i1 = ge ? OFF : OFF + 1;
        n.i2 = ge ? OFF + 1 : OFF;
        n.a3 = -INFINITY;
        n.s = n.a1 > -INFINITY ? 1.0f + __expf(n.a2 - n.a1) : 0.0f;
        return n;
    } else {
        const ChunkNode p = chunk_tree<OFF, N / 2>(r, v0, V, inv_temp);
        const ChunkNode q = chunk_tree<OFF + N / 2, N / 2>(r, v0, V, inv_temp);
        return chunk_merge(p, q);
    }
}

template <int EPI, int MT, int NB, int BN, int STAGES, int CL>
__global__ void __launch_bounds__(kThreads, 1)
tc_gemm_kernel(const __grid_constant__ CUtensorMap tmap_x, const __grid_constant__ CUtensorMap tmap_w0,
               const __grid_constant__ CUtensorMap tmap_w1, int n_rows, int K, int n_ntiles,
               int n_mgroups, int k_splits, int w_stream_once, EpiParams ep, int* status) {
    // Two kinds of cluster: kPair, a CTA pair on two M-tiles sharing each weight tile through
    // cta_group::2 MMAs; kSplitK, CL CTAs on the CL K-ranges of one output tile (one tile per
    // cluster), whose accumulators are summed through distributed shared memory.
    constexpr bool kSplitK = EPI == EPI_CGATEUP || EPI == EPI_CDOWN;
    constexpr bool kPair = CL > 1 && !kSplitK;
    using C = TileCfg<MT, NB, BN, STAGES, kPair>;
    static_assert(CL == 1 || kSplitK || (CL == 2 && NB == 1 && MT == 1), "a CTA pair shares one weight operand");
    static_assert(!kSplitK || (CL == 4 && MT == 2 && BN == 128), "cluster split-K: 4 K-ranges of a 256 x 128 tile");
    pdl_trigger();
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + STAGES * C::kStageBytes);
    uint64_t* empty = full + STAGES;
    uint64_t* tfull = empty + STAGES;
    uint64_t* tempty = tfull + 2;
    uint64_t* drain = tempty + 2;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
    volatile int* last_chunk = abort_flag + 1;   // [2]: this group's chunk was its unit's last

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    // Units are dealt to clusters. Pair: CTA `crank` of a cluster takes M-tile group member crank
    // of every unit. Split-K: a unit is an output tile and CTA crank takes K-range crank. With
    // CL = 1 a cluster is one CTA.
    const int n_units = kSplitK ? n_ntiles * n_mgroups : n_ntiles * n_mgroups * k_splits;
    const int crank = CL > 1 ? static_cast<int>(ptx::cluster_ctarank()) : 0;
    const int m_cl = kPair ? CL : 1, m_rank = kPair ? crank : 0;   // M-tiles of a cluster, this CTA's
    const bool leader = !kPair || crank == 0;                     // the pair's MMA issuer
    const int cid = CL > 1 ? static_cast<int>(ptx::cluster_id_x()) : static_cast<int>(blockIdx.x);
    const int ncl = CL > 1 ? static_cast<int>(ptx::cluster_count_x()) : static_cast<int>(gridDim.x);
    const int nk = K / kBK / k_splits;      // K-steps per unit (K % (64 * k_splits) == 0)
    const uint64_t wait_ns = ep.wait_ns ? ep.wait_ns : kWaitLimitNs;
    auto unit_of = [&](int u) {
        if constexpr (kSplitK) return Unit{u / n_mgroups, u % n_mgroups, crank};
        return decode_unit(u, n_mgroups, k_splits);
    };
    // Work items: the units, except that with a tail split each unit of the last round becomes
    // tail_split items over consecutive K-chunks of its range ([kb0, kb1) in K-steps).
    constexpr bool kTail = CL == 1 && (EPI == EPI_GATEUP || EPI == EPI_DOWN);
    const int n_split = kTail ? ep.tail_split : 0;
    const int n_items = n_split ? ep.n_full + (n_units - ep.n_full) * n_split : n_units;
    struct Item {
        Unit w;
        int kb0, kb1, tail, chunk;   // tail unit and chunk index (-1: a whole unit)
    };
    auto item_of = [&](int i) {
        Item it;
        const int ns = n_split > 0 ? n_split : 1;   // (a constant 1 in kernels without a tail split)
        if (n_split == 0 || i < ep.n_full) {
            it.w = unit_of(i);
            it.kb0 = it.w.kx * nk;
            it.kb1 = it.kb0 + nk;
            it.tail = it.chunk = -1;
        } else {
            const int r = i - ep.n_full;
            it.tail = r / ns;
            it.chunk = r - it.tail * ns;
            it.w = unit_of(ep.n_full + it.tail);
            it.kb0 = it.w.kx * nk + nk * it.chunk / ns;
            it.kb1 = it.w.kx * nk + nk * (it.chunk + 1) / ns;
        }
        return it;
    };
    // shared::cluster address of this CTA's barrier `bar` as seen at the same offset in the pair's
    // even CTA (pair mode: the barriers the issuer waits on) or in the odd one
    auto in_leader = [&](uint64_t* bar) {
        return kPair && crank != 0 ? ptx::mapa_shared(ptx::smem_u32(bar), 0) : ptx::smem_u32(bar);
    };
    auto in_peer = [&](uint64_t* bar) { return ptx::mapa_shared(ptx::smem_u32(bar), 1); };

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            ptx::mbar_init(&full[s], 1);
            ptx::mbar_init(&empty[s], 1);
        }
        for (int g = 0; g < 2; ++g) {
            ptx::mbar_init(&tfull[g], 1);
            // pair: one arrival per epilogue warp of both CTAs (used in the even CTA only)
            ptx::mbar_init(&tempty[g], kPair ? 2 * (kEpiWarps / 2) : 32 * kEpiWarps / 2);
        }
        ptx::mbar_init(drain, 1);
        *abort_flag = 0;
        ptx::fence_barrier_init();
    }
    if constexpr (kPair) {
        // both CTAs of the pair are running and their barriers exist before the collective
        // allocation and before either CTA signals the other's barriers
        ptx::cluster_sync();
        if (warp == 1) {
            ptx::tmem_alloc_pair(tmem_slot, 512);
            ptx::tmem_relinquish_pair();
        }
        ptx::tc_fence_before();
        __syncthreads();
        ptx::tc_fence_after();
    } else {
        if (warp == 1) {
            ptx::tmem_alloc(tmem_slot, 512);
            ptx::tmem_relinquish();
        }
        ptx::tc_fence_before();
        __syncthreads();
        if constexpr (CL > 1) ptx::cluster_sync();   // the peers' barriers exist before any remote access
        ptx::tc_fence_after();
    }
    const uint32_t tmem_base = *tmem_slot;
    if (!(warp == 0 && lane == 0)) pdl_wait();   // the producer waits after its weight prefetch
    // a call's status word starts at zero; cleared here, after every earlier kernel has finished,
    // instead of by a separate memset that would end the overlap with the previous kernel
    if (EPI == EPI_LMHEAD && ep.reset_status && blockIdx.x == 0 && threadIdx.x == 64 && status) *status = 0;

    if (warp == 0) {
        // ------------------------------------------------------------------ TMA producer
        if (lane == 0) {
            ptx::prefetch_tmap(&tmap_x);
            ptx::prefetch_tmap(&tmap_w0);
            if (NB == 2) ptx::prefetch_tmap(&tmap_w1);
            const uint64_t pol_x = ptx::policy_evict_last();
            const uint64_t pol_w = w_stream_once ? ptx::policy_evict_first() : ptx::policy_evict_last();
            // Pair: both CTAs' copies of a stage complete on the even CTA's full barrier, which
            // the even CTA alone arms with the bytes of both halves.
            constexpr uint32_t kTxBytes = (kPair ? 2 : 1) * C::kStageBytes;
            auto load_x = [&](uint8_t* sp, uint64_t* bar, int j, int kb, int mt) {
                if constexpr (kPair)
                    ptx::tma_load_2d_pair(sp + j * C::kABytes, &tmap_x, in_leader(bar), kb * kBK, mt * kBM, pol_x);
                else
                    ptx::tma_load_2d(sp + j * C::kABytes, &tmap_x, bar, kb * kBK, mt * kBM, pol_x);
            };
            // Weight tiles of one stage; in a pair each CTA stages its half of the rows
            // (tmap_w0's box is BN / 2 rows high).
            auto load_w = [&](uint8_t* sp, uint64_t* bar, int kb, int nt) {
                if constexpr (kPair) {
                    ptx::tma_load_2d_pair(sp + MT * C::kABytes, &tmap_w0, in_leader(bar), kb * kBK,
                                          nt * BN + crank * (BN / 2), pol_w);
                } else {
                    ptx::tma_load_2d(sp + MT * C::kABytes, &tmap_w0, bar, kb * kBK, nt * BN, pol_w);
                    if (NB == 2)
                        ptx::tma_load_2d(sp + MT * C::kABytes + C::kBBytes, &tmap_w1, bar, kb * kBK, nt * BN, pol_w);
                }
            };
            // The weights are no kernel's output: the first unit's first weight tiles are
            // requested before waiting for the previous kernel (which may be writing X).
            int pre = 0;
            if (cid < n_items) {
                const Item f = item_of(cid);
                pre = f.kb1 - f.kb0 < STAGES ? f.kb1 - f.kb0 : STAGES;
                for (int i = 0; i < pre; ++i) {
                    if (leader) ptx::mbar_arrive_expect_tx(&full[i], kTxBytes);
                    load_w(smem + i * C::kStageBytes, &full[i], f.kb0 + i, f.w.nt);
                }
            }
            pdl_wait();
            int stage = 0;
            uint32_t phase = 0;
            uint32_t issued_mask = 0;                 // stages that ever received a load
            uint32_t last_parity[STAGES > 0 ? STAGES : 1];
            bool ok = true;
            int it = 0;                               // k-steps issued so far by this CTA
            for (int u = cid; u < n_items && ok; u += ncl) {
                const Item itm = item_of(u);
                const int nt = itm.w.nt, mt0 = (itm.w.mg * m_cl + m_rank) * MT;
                for (int kb = itm.kb0; kb < itm.kb1; ++kb, ++it) {
                    if (!ptx::mbar_wait(&empty[stage], phase ^ 1u, abort_flag, wait_ns)) {
                        ok = false;
                        break;
                    }
                    uint8_t* sp = smem + stage * C::kStageBytes;
                    const bool w_done = it < pre;     // weight tiles already requested above
                    if (!w_done && leader) ptx::mbar_arrive_expect_tx(&full[stage], kTxBytes);
#pragma unroll
                    for (int j = 0; j < MT; ++j) load_x(sp, &full[stage], j, kb, mt0 + j);
                    if (!w_done) load_w(sp, &full[stage], kb, nt);
                    issued_mask |= 1u << stage;
                    last_parity[stage] = phase;
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
            if (!ok) {
                *abort_flag = 1;
                set_status(status, TF_DEV_TIMEOUT);
            }
            // No copy may still be writing this CTA's shared memory when it exits: wait for the
            // last load of every stage (already complete unless another role gave up early). The
            // odd CTA of a pair has no barrier of its own to wait on: its copies complete on the
            // even CTA's barriers, which the even CTA's producer waits for here before both CTAs
            // meet at the final cluster barrier; after giving up it waits a fixed 100 us, far
            // longer than any copy takes once issued.
            if (leader) {
                for (int s = 0; s < STAGES; ++s)
                    if (issued_mask & (1u << s)) ptx::mbar_wait(&full[s], last_parity[s], nullptr, kWaitLimitNs);
            } else if (!ok) {
                const uint64_t t0 = ptx::globaltimer_ns();
                while (ptx::globaltimer_ns() - t0 < 100000ull) {
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------------ MMA issuer
        if (lane == 0 && leader) {
            // the NB weight tiles of a stage are adjacent in shared memory with the same swizzle, so
            // one MMA of N = NB * BN covers them: A is read from shared memory once per k-step
            constexpr uint32_t kIdesc = ptx::idesc_bf16_f32(kPair ? 2 * kBM : kBM, NB * BN);
            int stage = 0;
            uint32_t phase = 0;
            uint32_t use[2] = {0u, 0u};
            bool ok = true;
            int kl = 0;
            for (int u = cid; u < n_items && ok; u += ncl, ++kl) {
                const int g0 = (MT == 2) ? 0 : (kl & 1);
                const Item itm = item_of(u);
                const int nk_u = itm.kb1 - itm.kb0;
                for (int j = 0; j < MT && ok; ++j)
                    ok = kPair ? ptx::mbar_wait_cluster(&tempty[g0 + j], (use[g0 + j] & 1u) ^ 1u, abort_flag, wait_ns)
                               : ptx::mbar_wait(&tempty[g0 + j], (use[g0 + j] & 1u) ^ 1u, abort_flag, wait_ns);
                if (!ok) break;
                ptx::tc_fence_after();
                for (int kb = 0; kb < nk_u; ++kb) {   // position inside the item's K range
                    const bool landed = kPair ? ptx::mbar_wait_cluster(&full[stage], phase, abort_flag, wait_ns)
                                              : ptx::mbar_wait(&full[stage], phase, abort_flag, wait_ns);
                    if (!landed) {
                        ok = false;
                        break;
                    }
                    ptx::tc_fence_after();
                    const uint32_t a0 = ptx::smem_u32(smem + stage * C::kStageBytes);
                    const uint32_t b0 = a0 + MT * C::kABytes;
#pragma unroll
                    for (int kk = 0; kk < kBK / 16; ++kk) {
                        const uint64_t bd = ptx::sw128_kmajor_desc(b0 + kk * 32);
#pragma unroll
                        for (int j = 0; j < MT; ++j) {
                            const uint64_t ad = ptx::sw128_kmajor_desc(a0 + j * C::kABytes + kk * 32);
                            const uint32_t acc = (kb | kk) != 0 ? 1u : 0u;
                            if constexpr (kPair)
                                ptx::mma_bf16_pair(tmem_base + 256u * (g0 + j), ad, bd, kIdesc, acc);
                            else
                                ptx::mma_bf16(tmem_base + 256u * (g0 + j), ad, bd, kIdesc, acc);
                        }
                    }
                    // frees the stage (in both CTAs of a pair) once these MMAs finish
                    if constexpr (kPair) {
                        ptx::mma_commit_pair(ptx::smem_u32(&empty[stage]));
                        ptx::mma_commit_pair(in_peer(&empty[stage]));
                    } else {
                        ptx::mma_commit(&empty[stage]);
                    }
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
                if (!ok) break;
                for (int j = 0; j < MT; ++j) {
                    if constexpr (kPair) {
                        ptx::mma_commit_pair(ptx::smem_u32(&tfull[g0 + j]));
                        ptx::mma_commit_pair(in_peer(&tfull[g0 + j]));
                    } else {
                        ptx::mma_commit(&tfull[g0 + j]);
                    }
                    ++use[g0 + j];
                }
            }
            if (!ok) {
                *abort_flag = 1;
                set_status(status, TF_DEV_TIMEOUT);
            }
            // every MMA issued so far must finish before TMEM is released
            if constexpr (kPair)
                ptx::mma_commit_pair(ptx::smem_u32(drain));
            else
                ptx::mma_commit(drain);
            ptx::mbar_wait(drain, 0, nullptr, kWaitLimitNs);
        }
    } else {
        // ------------------------------------------------------------------ epilogue
        const int e = warp - 2;
        const int g = e / (kEpiWarps / 2);          // accumulator slot of this group
        const int q = warp & 3;                     // TMEM lane quarter of this warp
        const int half = (e % (kEpiWarps / 2)) / 4; // which half of the columns this warp takes
        uint32_t use = 0;
        int kl = 0;
        // hands the accumulator slot back to the MMA issuer; in a pair one arrival per warp on
        // the even CTA's barrier, after the warp's TMEM loads have completed
        auto release_slot = [&](int slot) {
            ptx::tc_fence_before();
            if constexpr (kPair) {
                __syncwarp();
                if (lane == 0) ptx::mbar_arrive_cluster(in_leader(&tempty[slot]));
            } else {
                ptx::mbar_arrive(&tempty[slot]);
            }
        };
        for (int u = cid; u < n_items; u += ncl, ++kl) {
            if (MT == 1 && (kl & 1) != g) continue;
            if (!ptx::mbar_wait(&tfull[g], use & 1u, abort_flag, wait_ns)) {
                *abort_flag = 1;
                set_status(status, TF_DEV_TIMEOUT);
                break;
            }
            ++use;
            ptx::tc_fence_after();
            const Item itm = item_of(u);
            const Unit w = itm.w;
            const int nt = w.nt;
            const int row = ((w.mg * m_cl + m_rank) * MT + (MT == 2 ? g : 0)) * kBM + q * 32 + lane;
            const uint32_t tb = tmem_base + 256u * g + (static_cast<uint32_t>(q * 32) << 16);

            if (kTail && itm.chunk >= 0) {
                // ---- a K-chunk of a tail unit: its partial sums to `partial`; the group whose
                // chunk completes the unit's count adds all chunks in chunk order
                const int j = MT == 2 ? g : 0;                 // M-tile of the unit in this slot
                const int r = q * 32 + lane;                   // row within the M-tile
                constexpr int kUnitF4 = kBM * NB * BN / 4;     // float4s of one (chunk, M-tile)
                float4* part = reinterpret_cast<float4*>(ep.partial);
                auto at = [&](int ch, int col) {               // float4 of columns col..col+3, row r
                    return (static_cast<size_t>((itm.tail * n_split + ch) * MT + j) * kUnitF4) +
                           static_cast<size_t>(col >> 2) * kBM + r;
                };
#pragma unroll 1
                for (int nb = 0; nb < NB; ++nb) {
#pragma unroll 1
                    for (int c = half * (BN / 2); c < (half + 1) * (BN / 2); c += 32) {
                        uint32_t ra[32];
                        ptx::tmem_ld_32cols(tb + nb * BN + c, ra);
#pragma unroll
                        for (int f = 0; f < 8; ++f)
                            part[at(itm.chunk, nb * BN + c + 4 * f)] =
                                make_float4(__uint_as_float(ra[4 * f]), __uint_as_float(ra[4 * f + 1]),
                                            __uint_as_float(ra[4 * f + 2]), __uint_as_float(ra[4 * f + 3]));
                    }
                }
                release_slot(g);
                __threadfence();                                // this thread's partial sums, device-wide
                ptx::named_barrier_sync(1 + g, 32 * kEpiWarps / 2);
                if (e % (kEpiWarps / 2) == 0 && lane == 0) {
                    __threadfence();
                    const int done = atomicAdd(ep.sem + itm.tail * MT + j, 1);
                    last_chunk[g] = done == n_split - 1 ? 1 : 0;
                }
                ptx::named_barrier_sync(1 + g, 32 * kEpiWarps / 2);
                if (last_chunk[g]) {
                    __threadfence();                            // every chunk's partial sums
                    // 8 output columns at a time: this warp's half of the tile
#pragma unroll 1
                    for (int c = half * (BN / 2); c < (half + 1) * (BN / 2); c += 8) {
                        float a0[8], a1[8];
#pragma unroll
                        for (int t = 0; t < 8; ++t) a0[t] = a1[t] = 0.0f;
#pragma unroll 1
                        for (int ch = 0; ch < n_split; ++ch) {
                            const float4 p0 = part[at(ch, c)], p1 = part[at(ch, c + 4)];
                            a0[0] += p0.x; a0[1] += p0.y; a0[2] += p0.z; a0[3] += p0.w;
                            a0[4] += p1.x; a0[5] += p1.y; a0[6] += p1.z; a0[7] += p1.w;
                            if constexpr (NB == 2) {
                                const float4 u0 = part[at(ch, BN + c)], u1 = part[at(ch, BN + c + 4)];
                                a1[0] += u0.x; a1[1] += u0.y; a1[2] += u0.z; a1[3] += u0.w;
                                a1[4] += u1.x; a1[5] += u1.y; a1[6] += u1.z; a1[7] += u1.w;
                            }
                        }
                        if (row < n_rows) {
                            uint32_t o[4];
                            if constexpr (EPI == EPI_GATEUP) {
#pragma unroll
                                for (int t = 0; t < 4; ++t)
                                    o[t] = pack_bf16x2(silu_f(a0[2 * t]) * a1[2 * t], silu_f(a0[2 * t + 1]) * a1[2 * t + 1]);
                            } else {
                                const int sq = row / ep.R, rr = row - sq * ep.R;
                                const int hid_row = sq * ep.gamma + stage2_hidden_index(rr, ep.M);
                                const uint4 hv = *reinterpret_cast<const uint4*>(
                                    ep.hidden + static_cast<size_t>(hid_row) * ep.ld_out + nt * BN + c);
                                const uint32_t hw[4] = {hv.x, hv.y, hv.z, hv.w};
#pragma unroll
                                for (int t = 0; t < 4; ++t) {
                                    const __nv_bfloat162 h2 = *reinterpret_cast<const __nv_bfloat162*>(&hw[t]);
                                    o[t] = pack_bf16x2(__bfloat162float(h2.x) + a0[2 * t], __bfloat162float(h2.y) + a0[2 * t + 1]);
                                }
                            }
                            *reinterpret_cast<uint4*>(ep.out + static_cast<size_t>(row) * ep.ld_out + nt * BN + c) =
                                make_uint4(o[0], o[1], o[2], o[3]);
                        }
                    }
                    // the count starts from zero for the next call
                    ptx::named_barrier_sync(1 + g, 32 * kEpiWarps / 2);
                    if (e % (kEpiWarps / 2) == 0 && lane == 0) ep.sem[itm.tail * MT + j] = 0;
                }
            } else if constexpr (kSplitK) {
                // the accumulators are summed across the cluster below, once every CTA has them
            } else if constexpr (EPI == EPI_LMHEAD) {
                static_assert(BN == kBlockV, "one LM-head N tile is one vocabulary block");
                // this warp's half of the block: chunks [half * 4, half * 4 + 4)
                constexpr int kHalf = kChunks / 2;
                const Partials& P = ep.partials;
                // warps whose 32 rows are all padding skip the accumulators entirely
                if (row - lane < n_rows) {
                    float hm = -INFINITY, hsum = 0.0f, hbv = -INFINITY;
                    int hbid = -1;
                    // half summary; chunks arrive in id order, so strict > keeps the smaller id
                    auto fold = [&](const ChunkNode& c, int ci, int v0) {
                        if (c.a1 > hbv) {
                            hbv = c.a1;
                            hbid = v0 + c.i1;
                        }
                        if (c.a1 > -INFINITY) {
                            const float mn = fmaxf(hm, c.a1);
                            hsum = hsum * __expf(hm - mn) + c.s * __expf(c.a1 - mn);
                            hm = mn;
                        }
                        if (row < n_rows)
                            P.chunks[P.chunk_at(nt, ci, row)] =
                                make_float4(c.a1, c.a2, c.a3, __int_as_float(c.i1 | (c.i2 << 8)));
                    };
                    // Chunks in pairs: both TMEM loads in flight together, the two trees independent
                    // of each other (so their instructions interleave), and the next pair's loads
                    // issued before this pair is folded and stored.
                    const int cb = half * kHalf;
                    uint32_t ra[32], rb[32];
                    ptx::tmem_ld_32cols_nowait(tb + cb * kChunk, ra);
                    ptx::tmem_ld_32cols_nowait(tb + (cb + 1) * kChunk, rb);
                    ptx::tmem_wait_ld_regs(ra);
                    ptx::tmem_wait_ld_regs(rb);
#pragma unroll
                    for (int pr = 0; pr < kHalf / 2; ++pr) {
                        const int ci = cb + 2 * pr;
                        const int v0 = nt * BN + ci * kChunk;
                        const ChunkNode c0 = chunk_tree<0, 32>(ra, v0, ep.V, ep.inv_temp);
                        const ChunkNode c1 = chunk_tree<0, 32>(rb, v0 + kChunk, ep.V, ep.inv_temp);
                        const bool more = pr + 1 < kHalf / 2;
                        if (more) {
                            __syncwarp();   // converged for the warp-collective TMEM loads
                            ptx::tmem_ld_32cols_nowait(tb + (ci + 2) * kChunk, ra);
                            ptx::tmem_ld_32cols_nowait(tb + (ci + 3) * kChunk, rb);
                        }
                        fold(c0, ci, v0);
                        fold(c1, ci + 1, v0 + kChunk);
                        if (more) {
                            __syncwarp();
                            ptx::tmem_wait_ld_regs(ra);
                            ptx::tmem_wait_ld_regs(rb);
                        }
                    }
                    if (row < n_rows)
                        P.halves[P.half_at(nt, half, row)] = make_float4(hm, hsum, hbv, __int_as_float(hbid));
                }
                release_slot(g);
            } else if constexpr (EPI == EPI_PARTIAL) {
                // float4-major: each store instruction writes the warp's 32 rows of 4 columns, 512
                // contiguous bytes
                float4* split = reinterpret_cast<float4*>(ep.partial + static_cast<size_t>(w.kx) * ep.n_cols * n_rows);
#pragma unroll 1
                for (int nb = 0; nb < NB; ++nb) {
#pragma unroll 1
                    for (int c = half * (BN / 2); c < (half + 1) * (BN / 2); c += 32) {
                        uint32_t ra[32];
                        ptx::tmem_ld_32cols(tb + nb * BN + c, ra);
                        if (row < n_rows) {
                            const int col = nb * ep.n_total + nt * BN + c;
                            float4* dst = split + static_cast<size_t>(col >> 2) * n_rows + row;
#pragma unroll
                            for (int j = 0; j < 8; ++j)
                                dst[static_cast<size_t>(j) * n_rows] = make_float4(__uint_as_float(ra[4 * j]), __uint_as_float(ra[4 * j + 1]),
                                                     __uint_as_float(ra[4 * j + 2]), __uint_as_float(ra[4 * j + 3]));
                        }
                    }
                }
                release_slot(g);
            } else if constexpr (EPI == EPI_GATEUP) {
#pragma unroll 1
                for (int c = half * (BN / 2); c < (half + 1) * (BN / 2); c += 32) {
                    uint32_t rg[32], ru[32];
                    ptx::tmem_ld_32cols(tb + c, rg);
                    ptx::tmem_ld_32cols(tb + BN + c, ru);
                    uint32_t packed[16];
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        const float a0 = silu_f(__uint_as_float(rg[2 * j])) * __uint_as_float(ru[2 * j]);
                        const float a1 = silu_f(__uint_as_float(rg[2 * j + 1])) * __uint_as_float(ru[2 * j + 1]);
                        packed[j] = pack_bf16x2(a0, a1);
                    }
                    if (row < n_rows) {
                        uint4* dst = reinterpret_cast<uint4*>(ep.out + static_cast<size_t>(row) * ep.ld_out + nt * BN + c);
#pragma unroll
                        for (int j = 0; j < 4; ++j)
                            dst[j] = make_uint4(packed[4 * j], packed[4 * j + 1], packed[4 * j + 2], packed[4 * j + 3]);
                    }
                }
                release_slot(g);
            } else {  // EPI_DOWN
                int hid_row = 0;
                if (row < n_rows) {
                    const int sq = row / ep.R, rr = row - sq * ep.R;
                    hid_row = sq * ep.gamma + stage2_hidden_index(rr, ep.M);
                }
#pragma unroll 1
                for (int c = half * (BN / 2); c < (half + 1) * (BN / 2); c += 32) {
                    uint32_t ra[32];
                    ptx::tmem_ld_32cols(tb + c, ra);
                    if (row < n_rows) {
                        const uint4* res = reinterpret_cast<const uint4*>(
                            ep.hidden + static_cast<size_t>(hid_row) * ep.ld_out + nt * BN + c);
                        uint4* dst = reinterpret_cast<uint4*>(ep.out + static_cast<size_t>(row) * ep.ld_out + nt * BN + c);
#pragma unroll
                        for (int j = 0; j < 4; ++j) {
                            const uint4 hv = res[j];
                            const uint32_t hw[4] = {hv.x, hv.y, hv.z, hv.w};
                            uint32_t o[4];
#pragma unroll
                            for (int t = 0; t < 4; ++t) {
                                const __nv_bfloat162 h2 = *reinterpret_cast<const __nv_bfloat162*>(&hw[t]);
                                const float x0 = __bfloat162float(h2.x) + __uint_as_float(ra[8 * j + 2 * t]);
                                const float x1 = __bfloat162float(h2.y) + __uint_as_float(ra[8 * j + 2 * t + 1]);
                                o[t] = pack_bf16x2(x0, x1);
                            }
                            dst[j] = make_uint4(o[0], o[1], o[2], o[3]);
                        }
                    }
                }
                release_slot(g);
            }
        }
    }

    if constexpr (kSplitK) {
        // ------------------------------------------------------------------ split-K sum
        // The tile's output columns are owned in CL blocks of BN / CL: CTA o adds the CL partial
        // sums of block o in K-range order (the order of the split-K reduction kernels) and
        // applies the epilogue. Every CTA writes the blocks it does not own to the exchange area
        // in global memory (it stays in L2; through L2 this takes half the time of remote
        // shared-memory stores), laid out [cluster][owner][sender slot][16-byte unit][row] so that
        // the 32 lanes (rows) of a warp store and load 512 contiguous bytes; one cluster barrier
        // (release/acquire at cluster scope) then makes them visible to their owners.
        constexpr int kOwn = BN / CL;                    // output columns per owner
        constexpr int kRowF4 = NB * kOwn / 4;            // 16-byte units per row of a block
        constexpr int kSlotF4 = MT * kBM * kRowF4;       // 16-byte units of one block
        static_assert(kOwn == 32, "one TMEM load per block and accumulator");
        const bool has_unit = cid < n_units;
        const int e = warp - 2;
        const int g = e / (kEpiWarps / 2), q = warp & 3, half = (e % (kEpiWarps / 2)) / 4;
        const int r = g * kBM + q * 32 + lane;           // tile row: TMEM slot g, lane q * 32 + lane
        const uint32_t tb = tmem_base + 256u * g + (static_cast<uint32_t>(q * 32) << 16);
        float4* xchg = reinterpret_cast<float4*>(ep.partial);
        // (the epilogue warps waited for this CTA's accumulators in the loop above)
        if (warp >= 2 && has_unit) {
            // the warp's half of the columns holds the blocks of owners 2 half and 2 half + 1
            for (int o = 2 * half; o < 2 * half + 2; ++o) {
                if (o == crank) continue;
                const int slot = crank < o ? crank : crank - 1;
                float4* dst = xchg + (static_cast<size_t>(cid * CL + o) * (CL - 1) + slot) * kSlotF4 + r;
#pragma unroll
                for (int nb = 0; nb < NB; ++nb) {
                    uint32_t ra[32];
                    ptx::tmem_ld_32cols(tb + nb * BN + o * kOwn, ra);
#pragma unroll
                    for (int f = 0; f < 8; ++f)
                        dst[(nb * 8 + f) * (MT * kBM)] = make_float4(__uint_as_float(ra[4 * f]), __uint_as_float(ra[4 * f + 1]),
                                                                   __uint_as_float(ra[4 * f + 2]), __uint_as_float(ra[4 * f + 3]));
                }
            }
        }
        __syncwarp();
        ptx::tc_fence_before();
        ptx::cluster_sync();   // every block is in the exchange area
        ptx::tc_fence_after();
        if (warp >= 2 && has_unit) {
            // this warp: 16 of the own block's columns, c0 .. c0 + 15 of the tile
            const Unit w = unit_of(cid);
            const int c0 = crank * kOwn + half * 16;
            const int row = w.mg * MT * kBM + r;
            float acc[NB][16];
#pragma unroll
            for (int kx = 0; kx < CL; ++kx) {
#pragma unroll
                for (int nb = 0; nb < NB; ++nb) {
                    float v[16];
                    if (kx == crank) {
                        uint32_t ra[16];
                        ptx::tmem_ld_16cols(tb + nb * BN + c0, ra);
#pragma unroll
                        for (int j = 0; j < 16; ++j) v[j] = __uint_as_float(ra[j]);
                    } else {
                        const int slot = kx < crank ? kx : kx - 1;
                        const float4* src = xchg + (static_cast<size_t>(cid * CL + crank) * (CL - 1) + slot) * kSlotF4 + r;
#pragma unroll
                        for (int f = 0; f < 4; ++f) {
                            const float4 t = src[(nb * 8 + half * 4 + f) * (MT * kBM)];
                            v[4 * f] = t.x;
                            v[4 * f + 1] = t.y;
                            v[4 * f + 2] = t.z;
                            v[4 * f + 3] = t.w;
                        }
                    }
#pragma unroll
                    for (int j = 0; j < 16; ++j) acc[nb][j] = kx == 0 ? v[j] : acc[nb][j] + v[j];
                }
            }
            if (row < n_rows) {
                const size_t col = static_cast<size_t>(w.nt) * BN + c0;
                uint32_t packed[8];
                if constexpr (EPI == EPI_CGATEUP) {
#pragma unroll
                    for (int j = 0; j < 8; ++j)
                        packed[j] = pack_bf16x2(silu_f(acc[0][2 * j]) * acc[NB - 1][2 * j],
                                                silu_f(acc[0][2 * j + 1]) * acc[NB - 1][2 * j + 1]);
                } else {
                    const int sq = row / ep.R, rr = row - sq * ep.R;
                    const int hid_row = sq * ep.gamma + stage2_hidden_index(rr, ep.M);
                    const uint4* res = reinterpret_cast<const uint4*>(ep.hidden + static_cast<size_t>(hid_row) * ep.ld_out + col);
#pragma unroll
                    for (int j = 0; j < 2; ++j) {
                        const uint4 hv = res[j];
                        const uint32_t hw[4] = {hv.x, hv.y, hv.z, hv.w};
#pragma unroll
                        for (int t = 0; t < 4; ++t) {
                            const __nv_bfloat162 h2 = *reinterpret_cast<const __nv_bfloat162*>(&hw[t]);
                            packed[4 * j + t] = pack_bf16x2(__bfloat162float(h2.x) + acc[0][8 * j + 2 * t],
                                                            __bfloat162float(h2.y) + acc[0][8 * j + 2 * t + 1]);
                        }
                    }
                }
                uint4* dst = reinterpret_cast<uint4*>(ep.out + static_cast<size_t>(row) * ep.ld_out + col);
                dst[0] = make_uint4(packed[0], packed[1], packed[2], packed[3]);
                dst[1] = make_uint4(packed[4], packed[5], packed[6], packed[7]);
            }
        }
    }

    // the producer and MMA lanes rejoin their warps first: the CTA-wide barrier below must wait
    // for every thread, not only for each warp's first arrivals
    __syncwarp();
    ptx::tc_fence_before();
    __syncthreads();
    // no CTA of the cluster may still write into this CTA's shared memory or barriers
    if constexpr (CL > 1) ptx::cluster_sync();
    if (warp == 1) {
        __syncwarp();
        ptx::tc_fence_after();
        if constexpr (kPair)
            ptx::tmem_dealloc_pair(tmem_base, 512);
        else
            ptx::tmem_dealloc(tmem_base, 512);
    }
}

// ------------------------------------------------------------------------------ host side

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) !=
                cudaSuccess ||
            q != cudaDriverEntryPointSuccess)
            p = nullptr;
        return reinterpret_cast<EncodeTiledFn>(p);
    }();
    return fn;
}

// Row-major bf16 matrix [outer, inner] read in boxes of box_inner x box_outer with 128B swizzle.
cudaError_t make_tmap(CUtensorMap* map, const void* base, uint64_t inner, uint64_t outer, uint32_t box_inner,
                      uint32_t box_outer) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return cudaErrorNotSupported;
    const cuuint64_t dims[2] = {inner, outer};
    const cuuint64_t strides[1] = {inner * 2};
    const cuuint32_t box[2] = {box_inner, box_outer};
    const cuuint32_t es[2] = {1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

// Clusters of CL CTAs that can be resident at once for this kernel (at most num_sms / CL).
template <typename K>
int resident_clusters(K kern, int smem, int cl, int num_sms) {
    int cap = num_sms / cl;
    if (cl == 1) return cap;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(cl * cap);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = cl;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess || n < 1) {
        (void)cudaGetLastError();
        return cap;
    }
    return n < cap ? n : cap;
}

template <int EPI, int MT, int NB, int BN, int STAGES, int CL = 1>
cudaError_t run_gemm(const Ctx& ctx, const CUtensorMap& tx, const CUtensorMap& tw0, const CUtensorMap& tw1,
                     int n_rows, int K, int n_ntiles, int n_mgroups, const EpiParams& ep_in, int k_splits = 1,
                     size_t partial_bytes = 0) {
    using C = TileCfg<MT, NB, BN, STAGES, (CL == 2 && EPI != EPI_CGATEUP && EPI != EPI_CDOWN)>;
    auto kern = tc_gemm_kernel<EPI, MT, NB, BN, STAGES, CL>;
    EpiParams ep = ep_in;
    ep.wait_ns = wait_limit_ns();
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes);
    if (e != cudaSuccess) return e;
    const int n_units = n_ntiles * n_mgroups * k_splits;
    const int stream_once = n_mgroups == 1 ? 1 : 0;
    if constexpr (EPI == EPI_CGATEUP || EPI == EPI_CDOWN) {
        // one output tile per cluster, its K-ranges on the cluster's CTAs; the caller has checked
        // that all clusters are resident at once (splitk_clusters_fit)
        e = launch_pdl_cluster(kern, dim3(CL * n_ntiles * n_mgroups), dim3(kThreads), C::kSmemBytes, ctx.stream, CL,
                               tx, tw0, tw1, n_rows, K, n_ntiles, n_mgroups, CL, stream_once, ep, ctx.status);
    } else if constexpr (CL == 1) {
        int n_items = n_units;
        if constexpr (EPI == EPI_GATEUP || EPI == EPI_DOWN) {
            // Tail split: when the units overflow the SMs by a last round that would leave most of
            // them idle, each unit of that round runs as up to kMaxTailSplit K-chunks on the idle
            // SMs, summed by the chunk that finishes last (fp32 partial sums in the workspace).
            const int tail = n_units % ctx.num_sms;
            int split = tail > 0 ? ctx.num_sms / tail : 0;
            split = split < kMaxTailSplit ? split : kMaxTailSplit;
            split = split < K / kBK ? split : K / kBK;
            const size_t need = static_cast<size_t>(tail) * split * MT * kBM * NB * BN * sizeof(float);
            if (k_splits == 1 && n_units > ctx.num_sms && split >= 2 && ctx.status && tail * MT <= kTailSems &&
                ep.partial && need <= partial_bytes) {
                ep.n_full = n_units - tail;
                ep.tail_split = split;
                ep.sem = ctx.status + 1;
                n_items = ep.n_full + tail * split;
            }
        }
        const int grid = n_items < ctx.num_sms ? n_items : ctx.num_sms;
        e = launch_pdl(kern, dim3(grid), dim3(kThreads), C::kSmemBytes, ctx.stream, tx, tw0, tw1, n_rows, K,
                       n_ntiles, n_mgroups, k_splits, stream_once, ep, ctx.status);
    } else {
        static const int max_cl = resident_clusters(kern, C::kSmemBytes, CL, ctx.num_sms);
        const int n_cl = n_units < max_cl ? n_units : max_cl;
        e = launch_pdl_cluster(kern, dim3(CL * n_cl), dim3(kThreads), C::kSmemBytes, ctx.stream, CL, tx, tw0, tw1,
                               n_rows, K, n_ntiles, n_mgroups, k_splits, stream_once, ep, ctx.status);
    }
    return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace

// Bytes of the split-K exchange area of the cluster path: per output tile (cluster) of 128
// columns, CL = 4 owners receive 3 blocks of 2 M-tiles x 128 rows x NB x 32 fp32 columns.
size_t splitk_exchange_bytes(int n_out_cols, int nb) {
    return static_cast<size_t>(n_out_cols / 128) * 4 * 3 * (2 * 128) * nb * 32 * 4;
}

namespace {

// Whether n_tiles clusters of the split-K kernel can all be resident at once (each cluster then
// runs its one tile; a second wave would serialise them).
template <int EPI, int MT, int NB, int BN, int STAGES, int CL>
bool splitk_clusters_fit(const Ctx& ctx, int n_tiles) {
    using C = TileCfg<MT, NB, BN, STAGES>;
    auto kern = tc_gemm_kernel<EPI, MT, NB, BN, STAGES, CL>;
    static const int max_cl = [&] {
        if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes) != cudaSuccess) {
            (void)cudaGetLastError();
            return 0;
        }
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(CL * (ctx.num_sms / CL));
        cfg.blockDim = dim3(kThreads);
        cfg.dynamicSmemBytes = C::kSmemBytes;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = CL;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        int n = 0;
        if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess) {
            (void)cudaGetLastError();
            return 0;
        }
        return n;
    }();
    return n_tiles <= max_cl;
}

}  // namespace

cudaError_t launch_lmhead_tc(const Ctx& ctx, const void* lm_head, const void* x, int n_rows, int d, int V,
                             float inv_temp, Partials partials, bool reset_status) {
    if (n_rows <= 0) return cudaSuccess;
    const int n_tiles = (V + kBlockV - 1) / kBlockV;
    const int m_tiles = (n_rows + kBM - 1) / kBM;
    // More than one M-tile: CTA pairs (clusters of two), one M-tile each, share every weight tile
    // through cta_group::2 MMAs (each stages half of its rows), so W_lm is read once while each
    // CTA keeps one TMEM slot per unit and overlaps its epilogue with the next unit's MMAs; 32 KB
    // per CTA and stage leaves room for seven stages.
    const int cl = m_tiles == 1 ? 1 : 2;
    CUtensorMap tx, tw;
    cudaError_t e = make_tmap(&tx, x, d, n_rows, kBK, kBM);
    if (e == cudaSuccess) e = make_tmap(&tw, lm_head, d, V, kBK, kBlockV / cl);
    if (e != cudaSuccess) return e;
    EpiParams ep{};
    ep.partials = partials;
    ep.V = V;
    ep.inv_temp = inv_temp;
    ep.reset_status = reset_status ? 1 : 0;
    if (m_tiles == 1) return run_gemm<EPI_LMHEAD, 1, 1, kBlockV, 4>(ctx, tx, tw, tw, n_rows, d, n_tiles, 1, ep);
    return run_gemm<EPI_LMHEAD, 1, 1, kBlockV, 7, 2>(ctx, tx, tw, tw, n_rows, d, n_tiles, (m_tiles + 1) / 2, ep);
}

// Split-K factor for a GEMM with `base_units` (N tiles x M-tile groups) and nk K-steps: enough
// units to cover the SMs, at most kMaxKSplits, and a divisor of nk.
int choose_k_splits(int base_units, int nk, int num_sms) {
    int ks = base_units >= num_sms ? 1 : num_sms / base_units;
    if (ks > kMaxKSplits) ks = kMaxKSplits;
    while (ks > 1 && nk % ks != 0) --ks;
    return ks < 1 ? 1 : ks;
}

// h' = h + In W^T with In [n_rows, K] (tmap_in, boxes of kBK x kBM) and W [d, K] (tmap_w, boxes of
// kBK x BN, BN = 128 when d % 128 == 0, else 64): the SwiGLU down projection (K = I, In = A) and
// the linear approximator (K = 2d, In = x). The residual row of stage-2 row r is the hidden state
// of its depth; the epilogue adds it in fp32 and rounds once to bf16.
static cudaError_t run_residual_gemm(const Ctx& ctx, const CUtensorMap& ta, const CUtensorMap& td, int K, const void* hidden,
                              int n_rows, int d, int R, int M, int gamma, void* h_prime, float* partial,
                              size_t partial_bytes) {
    constexpr int BN = 128;
    const int m_tiles = (n_rows + kBM - 1) / kBM;
    const int n_mg = m_tiles == 1 ? 1 : (m_tiles + 1) / 2;
    const int bn_d = d % BN == 0 ? BN : 64;
    const int ks2 = choose_k_splits((d / bn_d) * n_mg, K / kBK, ctx.num_sms);
    EpiParams ed{};
    ed.out = static_cast<__nv_bfloat16*>(h_prime);
    ed.ld_out = d;
    ed.hidden = static_cast<const __nv_bfloat16*>(hidden);
    ed.R = R;
    ed.M = M;
    ed.gamma = gamma;
    ed.partial = partial;
    ed.n_cols = d;
    ed.n_total = d;
    if (ks2 == 1) {
        if (bn_d == BN)
            return m_tiles == 1 ? run_gemm<EPI_DOWN, 1, 1, BN, 6>(ctx, ta, td, td, n_rows, K, d / BN, 1, ed, 1, partial_bytes)
                                : run_gemm<EPI_DOWN, 2, 1, BN, 4>(ctx, ta, td, td, n_rows, K, d / BN, n_mg, ed, 1, partial_bytes);
        return m_tiles == 1 ? run_gemm<EPI_DOWN, 1, 1, 64, 8>(ctx, ta, td, td, n_rows, K, d / 64, 1, ed, 1, partial_bytes)
                            : run_gemm<EPI_DOWN, 2, 1, 64, 5>(ctx, ta, td, td, n_rows, K, d / 64, n_mg, ed, 1, partial_bytes);
    }
    if (m_tiles == 2 && bn_d == BN && ks2 == 4 && splitk_clusters_fit<EPI_CDOWN, 2, 1, BN, 4, 4>(ctx, d / BN))
        return run_gemm<EPI_CDOWN, 2, 1, BN, 4, 4>(ctx, ta, td, td, n_rows, K, d / BN, 1, ed, 4);
    cudaError_t e;
    if (bn_d == BN)
        e = m_tiles == 1 ? run_gemm<EPI_PARTIAL, 1, 1, BN, 6>(ctx, ta, td, td, n_rows, K, d / BN, 1, ed, ks2)
                         : run_gemm<EPI_PARTIAL, 2, 1, BN, 4>(ctx, ta, td, td, n_rows, K, d / BN, n_mg, ed, ks2);
    else
        e = m_tiles == 1 ? run_gemm<EPI_PARTIAL, 1, 1, 64, 8>(ctx, ta, td, td, n_rows, K, d / 64, 1, ed, ks2)
                         : run_gemm<EPI_PARTIAL, 2, 1, 64, 5>(ctx, ta, td, td, n_rows, K, d / 64, n_mg, ed, ks2);
    if (e != cudaSuccess) return e;
    return launch_down_reduce(ctx, partial, ks2, n_rows, d, static_cast<const __nv_bfloat16*>(hidden), R, M, gamma,
                              static_cast<__nv_bfloat16*>(h_prime));
}

cudaError_t launch_swiglu_tc(const Ctx& ctx, const void* X, int k_in, const void* w_gate, const void* w_up,
                             const void* w_down, const void* hidden, int n_rows, int d, int I, int R, int M,
                             int gamma, void* A, void* h_prime, float* partial, size_t partial_bytes) {
    if (n_rows <= 0) return cudaSuccess;
    constexpr int BN = 128;
    const int m_tiles = (n_rows + kBM - 1) / kBM;
    const int n_mg = m_tiles == 1 ? 1 : (m_tiles + 1) / 2;
    const int bn_gu = I % BN == 0 ? BN : 64;
    const int bn_d = d % BN == 0 ? BN : 64;
    CUtensorMap tx, tg, tu, ta, td;
    cudaError_t e = make_tmap(&tx, X, k_in, n_rows, kBK, kBM);
    if (e == cudaSuccess) e = make_tmap(&tg, w_gate, k_in, I, kBK, bn_gu);
    if (e == cudaSuccess) e = make_tmap(&tu, w_up, k_in, I, kBK, bn_gu);
    if (e == cudaSuccess) e = make_tmap(&ta, A, I, n_rows, kBK, kBM);
    if (e == cudaSuccess) e = make_tmap(&td, w_down, I, d, kBK, bn_d);
    if (e != cudaSuccess) return e;

    // ---- gate/up: A = SiLU(X Wg^T) * (X Wu^T)
    const int ks1 = choose_k_splits((I / bn_gu) * n_mg, k_in / kBK, ctx.num_sms);
    EpiParams ep{};
    ep.out = static_cast<__nv_bfloat16*>(A);
    ep.ld_out = I;
    ep.partial = partial;
    ep.n_cols = 2 * I;
    ep.n_total = I;
    if (ks1 == 1) {
        if (bn_gu == BN)
            e = m_tiles == 1 ? run_gemm<EPI_GATEUP, 1, 2, BN, 4>(ctx, tx, tg, tu, n_rows, k_in, I / BN, 1, ep, 1, partial_bytes)
                             : run_gemm<EPI_GATEUP, 2, 2, BN, 3>(ctx, tx, tg, tu, n_rows, k_in, I / BN, n_mg, ep, 1, partial_bytes);
        else
            e = m_tiles == 1 ? run_gemm<EPI_GATEUP, 1, 2, 64, 6>(ctx, tx, tg, tu, n_rows, k_in, I / 64, 1, ep, 1, partial_bytes)
                             : run_gemm<EPI_GATEUP, 2, 2, 64, 4>(ctx, tx, tg, tu, n_rows, k_in, I / 64, n_mg, ep, 1, partial_bytes);
        if (e != cudaSuccess) return e;
    } else if (m_tiles == 2 && bn_gu == BN && ks1 == 4 &&
               splitk_clusters_fit<EPI_CGATEUP, 2, 2, BN, 3, 4>(ctx, I / BN)) {
        e = run_gemm<EPI_CGATEUP, 2, 2, BN, 3, 4>(ctx, tx, tg, tu, n_rows, k_in, I / BN, 1, ep, 4);
        if (e != cudaSuccess) return e;
    } else {
        if (bn_gu == BN)
            e = m_tiles == 1 ? run_gemm<EPI_PARTIAL, 1, 2, BN, 4>(ctx, tx, tg, tu, n_rows, k_in, I / BN, 1, ep, ks1)
                             : run_gemm<EPI_PARTIAL, 2, 2, BN, 3>(ctx, tx, tg, tu, n_rows, k_in, I / BN, n_mg, ep, ks1);
        else
            e = m_tiles == 1 ? run_gemm<EPI_PARTIAL, 1, 2, 64, 6>(ctx, tx, tg, tu, n_rows, k_in, I / 64, 1, ep, ks1)
                             : run_gemm<EPI_PARTIAL, 2, 2, 64, 4>(ctx, tx, tg, tu, n_rows, k_in, I / 64, n_mg, ep, ks1);
        if (e != cudaSuccess) return e;
        e = launch_swiglu_reduce(ctx, partial, ks1, n_rows, I, static_cast<__nv_bfloat16*>(A));
        if (e != cudaSuccess) return e;
    }

    // ---- down + residual: h' = h + A Wd^T
    return run_residual_gemm(ctx, ta, td, I, hidden, n_rows, d, R, M, gamma, h_prime, partial, partial_bytes);
}

cudaError_t launch_linear_tc(const Ctx& ctx, const void* X, const void* w_lin, const void* hidden, int n_rows, int d,
                             int R, int M, int gamma, void* h_prime, float* partial, size_t partial_bytes) {
    if (n_rows <= 0) return cudaSuccess;
    const int bn = d % 128 == 0 ? 128 : 64;
    CUtensorMap tx, tw;
    cudaError_t e = make_tmap(&tx, X, 2 * d, n_rows, kBK, kBM);
    if (e == cudaSuccess) e = make_tmap(&tw, w_lin, 2 * d, d, kBK, bn);
    if (e != cudaSuccess) return e;
    return run_residual_gemm(ctx, tx, tw, 2 * d, hidden, n_rows, d, R, M, gamma, h_prime, partial, partial_bytes);
}

}  // namespace tf
