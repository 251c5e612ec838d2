"""GPU parity: the CUDA path through the C ABI against the fp64 oracle on the same seeded inputs.

fp32 inputs: every log-probability within 1e-4 of the plain fp64 oracle, tree structure
bit-exact wherever the oracle's order margin exceeds 1e-3.
bf16 inputs with fp32 accumulation (tests/parity.py, BF16): each stage against the oracle's
formula on the GPU's own inputs to that stage -- x correctly rounded; SiLU(G)*U and h' within one
bf16 ulp plus the fp32 accumulation error; the LM head's log-probabilities of the GPU's h' within
1e-3; the tree equal to the oracle's Part 2 run on the GPU's lists -- and end to end: stage 1
within 1e-3 of the plain oracle; stage 2 within 0.1 and node scores within 0.06 of the oracle
that rounds to bf16 where the GPU stores bf16; the tree's structure against that oracle's at
every cut of its pop order that the node bound decides (bit-exact over the decided prefix).
"""
import numpy as np
import pytest
import torch

import synth
from oracle import treeflash_oracle as O

pytestmark = pytest.mark.gpu

import parity  # noqa: E402  (tests/ is on sys.path)


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_03819_gb300 import binding
    if not __import__("os").path.exists(binding.LIB_PATH):
        from paper_2606_03819_gb300 import build
        build.build()
    binding.load_library()


def check(cfg, emulate_also=True, inp=None, orc_seqs=None, W=None):
    """fp32: everything against the plain fp64 oracle (1e-4, structure exact beyond 1e-3).
    bf16: every stage against the oracle's formula on the GPU's own inputs, then end to end
    (tests/parity.py explains the bounds). W: the oracle's weights, if already widened."""
    inp = inp if inp is not None else synth.make_inputs(cfg)
    dinp = parity.device_inputs(inp)
    gpu = parity.run_gpu(cfg, dinp)
    W = W if W is not None else parity.oracle_weights(inp)
    reps = {}
    seqs = list(range(cfg.batch)) if orc_seqs is None else orc_seqs
    sub = {k: (v[seqs] if isinstance(v, np.ndarray) and v.ndim >= 1 and v.shape[0] == cfg.batch else v)
           for k, v in gpu.items()}
    orc = parity.run_oracle(cfg, inp, emulate_bf16=False, seqs=seqs, W=W)
    if cfg.dtype == "f32":
        tol = parity.TOLS["f32"]
        reps["pure"] = parity.compare(cfg, sub, orc, tol["lp"], tol["sel"])
    else:
        orc_e = parity.run_oracle(cfg, inp, emulate_bf16=True, seqs=seqs, W=W) if cfg.mode == "ar" else None
        reps["e2e"] = parity.check_bf16_end_to_end(cfg, sub, orc, orc_e)
        if cfg.mode == "ar" and orc_seqs is None:
            reps["stagewise"] = parity.check_bf16_stagewise(cfg, inp, W, gpu)
    assert not (gpu["flags"] & ~16), f"device flags {gpu['flags']}"
    return gpu, reps


# ------------------------------------------------------------------ fp32 (CUDA-core) path


@pytest.mark.parametrize("name", ["tiny_f32", "tiny_peaked"])
def test_fp32_tiny(name):
    _, reps = check(synth.get_config(name))
    print(reps)


@pytest.mark.parametrize("mode", ["marginal", "marginal_mary"])
def test_fp32_marginal_modes(mode):
    check(synth.get_config("tiny_peaked", mode=mode))


def test_fp32_brute_force_v16():
    cfg = synth.get_config("tiny_v16", h_entropy=(1.0, 1.5), wd_std=0.5)
    gpu, _ = check(cfg)
    inp = synth.make_inputs(cfg)
    o = parity.run_oracle(cfg, inp)[0]
    src = O.ChildSource("ar", cfg.gamma, cfg.M, o.top_ids, o.s1_logp, o.s2_logp)
    uni = sorted(O.eligible_universe(src), key=lambda x: (-x[0], x[1]))
    best = {p for _, _, p in uni[: cfg.B]}
    assert parity._paths(gpu["node_tok"][0], gpu["node_parent"][0]) == best


# ------------------------------------------------------------------ bf16 (tcgen05) path

BF16_SMALL = [
    # (batch, V, gamma, M, K2, B): stage-1 rows b*gamma, stage-2 rows b*(1+M(gamma-1))
    (2, 2000, 4, 4, 12, 12),     # 8 / 26 rows: one M-tile, ragged last vocabulary block
    (12, 2304, 4, 4, 12, 12),    # 48 / 156 rows: two M-tiles in one unit
    (24, 2049, 4, 4, 12, 12),    # 96 / 312 rows: three M-tiles (half-empty last group), V = 8*256+1
    (40, 1536, 4, 4, 8, 16),     # 160 / 520 rows: two M-tiles already in stage 1; K2 < B
]


@pytest.mark.parametrize("b,V,gamma,M,K2,B", BF16_SMALL)
def test_bf16_small(b, V, gamma, M, K2, B):
    cfg = synth.get_config("tiny_peaked", dtype="bf16", batch=b, V=V, gamma=gamma, M=M, K2=K2, B=B)
    _, reps = check(cfg)
    print(reps)


def test_bf16_d_and_I_several_k_blocks():
    # d = 320 (5 K-steps of 64), I = 192 (3 N-tiles of 64 in the MLP), gamma 5, M 3
    cfg = synth.get_config("tiny_peaked", dtype="bf16", batch=3, d=320, I=192, V=3000, gamma=5, M=3,
                           K2=16, B=16)
    check(cfg)


def test_bf16_two_m_tiles_cluster_split_k():
    # 1 + M(gamma - 1) = 241 stage-2 rows (two 128-row tiles) with d = I = 512: both approximator
    # GEMMs split K over 4-CTA clusters and add the partial sums in distributed shared memory
    cfg = synth.get_config("tiny_peaked", dtype="bf16", batch=1, d=512, I=512, V=3000, gamma=16, M=16,
                           K2=16, B=32)
    check(cfg)


def test_bf16_tail_split_of_the_last_round():
    # 150 sequences x 13 rows = 1950 stage-2 rows (8 pairs of M-tiles) with d = I = 2560: on 152
    # SMs both approximator GEMMs have 20 x 8 = 160 work units, so the 8 units of the last round
    # run as 8 K-chunks each, added by the chunk that finishes last. Every stage is checked on
    # every row, the tree end to end on three sequences, and a second call on the same workspace
    # (its counters reset by the first) gives the same bits.
    from paper_2606_03819_gb300 import Dims, Drafter
    cfg = synth.get_config("tiny_peaked", dtype="bf16", batch=150, d=2560, I=2560, V=2000, wd_std=0.05)
    inp = synth.make_inputs(cfg)
    dinp = parity.device_inputs(inp)
    dr = Drafter(Dims.from_config(cfg), dinp)
    gpu = parity.run_gpu(cfg, dinp, drafter=dr)
    assert not (gpu["flags"] & ~16), f"device flags {gpu['flags']}"
    W = parity.oracle_weights(inp)
    parity.check_bf16_stagewise(cfg, inp, W, gpu)
    seqs = [0, 77, 149]
    sub = {k: (v[seqs] if isinstance(v, np.ndarray) and v.ndim >= 1 and v.shape[0] == cfg.batch else v)
           for k, v in gpu.items()}
    orc = parity.run_oracle(cfg, inp, seqs=seqs, W=W)
    orc_e = parity.run_oracle(cfg, inp, emulate_bf16=True, seqs=seqs, W=W)
    parity.check_bf16_end_to_end(cfg, sub, orc, orc_e)
    again = parity.run_gpu(cfg, dinp, drafter=dr)
    for k in ("A", "hp", "child_ids", "child_logp", "node_tok", "node_parent", "mask"):
        np.testing.assert_array_equal(gpu[k], again[k], err_msg=k)


@pytest.mark.parametrize("mode", ["marginal", "marginal_mary"])
def test_bf16_marginal_modes(mode):
    check(synth.get_config("tiny_peaked", dtype="bf16", batch=3, V=2000, mode=mode))


def test_bf16_zero_approximator_equals_mary_marginal_tree():
    # W_down = 0 gives h' = h exactly, so TreeFlash's tree is the M-ary marginal tree
    from paper_2606_03819_gb300 import Dims
    cfg = synth.get_config("tiny_peaked", dtype="bf16", batch=4, V=2000)
    inp = synth.make_inputs(cfg)
    inp["w_down"].zero_()
    d = parity.device_inputs(inp)
    a = parity.run_gpu(cfg, d)
    b = parity.run_gpu(cfg.replace(mode="marginal_mary"), d)
    for k in ("node_tok", "node_parent", "node_depth", "mask", "pos_ids"):
        np.testing.assert_array_equal(a[k], b[k], err_msg=k)
    np.testing.assert_array_equal(a["node_score"], b["node_score"])


def test_bf16_batch_equals_single_sequences():
    cfg = synth.get_config("tiny_peaked", dtype="bf16", batch=5, V=2000)
    inp = synth.make_inputs(cfg)
    full = parity.run_gpu(cfg, parity.device_inputs(inp))
    one = cfg.replace(batch=1)
    for s in range(cfg.batch):
        sub = dict(inp)
        for k in ("hidden", "root_tok", "root_pos"):
            sub[k] = inp[k][s:s + 1].contiguous()
        r = parity.run_gpu(one, parity.device_inputs(sub))
        for k in ("top_ids", "top_logp", "child_ids", "child_logp", "node_tok", "node_parent", "node_score",
                  "mask", "pos_ids"):
            np.testing.assert_array_equal(r[k][0], full[k][s], err_msg=f"{k} seq {s}")


def test_bf16_recompute_path_is_exact():
    # 80 vocabulary rows of one 256-block aligned with every hidden state: the top-64 of each row
    # all sit in that block, so its 32-column chunks each hold more members of the top 64 than
    # their two kept candidates; certification must flag and recompute them
    cfg = synth.get_config("tiny_peaked", dtype="bf16", batch=1, V=4096, K2=64, B=64, M=4)
    inp = synth.make_inputs(cfg)
    g = torch.Generator().manual_seed(5)
    dirn = inp["hidden"][0].float().mean(0)
    W = inp["lm_head"].float()
    W[512:592] = dirn / dirn.norm() * (0.2 + 0.05 * torch.rand(80, 1, generator=g))
    inp["lm_head"] = W.to(torch.bfloat16)
    gpu = parity.run_gpu(cfg, parity.device_inputs(inp))
    assert gpu["flags"] & 16, "the certification should have triggered a recompute"
    parity.check_bf16_stagewise(cfg, inp, parity.oracle_weights(inp), gpu)


def test_host_path_matches_device_path():
    from paper_2606_03819_gb300 import Dims, alloc_workspace, binding
    cfg = synth.get_config("tiny_peaked", dtype="bf16", batch=3, V=2000)
    inp = synth.make_inputs(cfg)
    d = parity.device_inputs(inp)
    dev = parity.run_gpu(cfg, d)
    dims = Dims.from_config(cfg)
    ws = alloc_workspace(dims)
    n = cfg.B + 1
    pin = lambda t: t.pin_memory()
    out = dict(node_tok=torch.empty(cfg.batch, n, dtype=torch.int32), node_parent=torch.empty(cfg.batch, n, dtype=torch.int32),
               node_depth=torch.empty(cfg.batch, n, dtype=torch.int32), node_score=torch.empty(cfg.batch, n),
               mask=torch.empty(cfg.batch, n, n, dtype=torch.uint8), pos_ids=torch.empty(cfg.batch, n, dtype=torch.int32),
               dev_status=torch.empty(cfg.batch, dtype=torch.int32))
    out = {k: pin(v) for k, v in out.items()}
    st = binding.tf_draft_tree_host(dims, d, pin(inp["hidden"]), pin(inp["root_tok"]), pin(inp["root_pos"]),
                                    out["node_tok"], out["node_parent"], out["node_depth"], out["node_score"],
                                    out["mask"], out["pos_ids"], out["dev_status"], ws)
    assert st == 0
    for k in ("node_tok", "node_parent", "node_depth", "node_score", "mask", "pos_ids"):
        np.testing.assert_array_equal(out[k].numpy(), dev[k], err_msg=k)


def test_bad_root_token_is_flagged_not_fatal():
    cfg = synth.get_config("tiny_peaked", dtype="bf16", batch=2, V=2000)
    inp = synth.make_inputs(cfg)
    inp["root_tok"][1] = cfg.V + 7
    gpu = parity.run_gpu(cfg, parity.device_inputs(inp))
    assert gpu["flags"] & 1
    assert gpu["dev_status"][1] & 1 and not gpu["dev_status"][0] & 1


def test_underfull_universe_is_flagged():
    cfg = synth.get_config("tiny_peaked", gamma=1, M=2, K2=4, B=8)
    inp = synth.make_inputs(cfg)
    gpu = parity.run_gpu(cfg, parity.device_inputs(inp))
    assert gpu["dev_status"][0] & 2
    assert (gpu["node_parent"][0, 5:] == -1).all() and (gpu["node_tok"][0, 5:] == -1).all()
    assert gpu["mask"][0, 5:].sum() == 0 and gpu["mask"][0, :, 5:].sum() == 0
    orc = parity.run_oracle(cfg, inp)
    assert orc[0].tree.underfull
    np.testing.assert_array_equal(gpu["node_tok"][0], orc[0].tree.tok)


# ------------------------------------------------------------------ "w/ Linear" approximator
# (Sec. 4 "Model Design", Table 3): h' = h + W_lin [h~ ; e]. The same gather and normalisation,
# then one residual GEMM with K = 2d (fp32: the CUDA-core kernel; bf16: the tcgen05 kernel, with
# split-K over 4-CTA clusters for 129..256 rows).


def test_fp32_linear_approximator():
    _, reps = check(synth.get_config("tiny_peaked", approx="linear"))
    print(reps)


@pytest.mark.parametrize("b,V,gamma,M,K2,B", [BF16_SMALL[0], BF16_SMALL[1], BF16_SMALL[2]])
def test_bf16_linear_approximator_small(b, V, gamma, M, K2, B):
    cfg = synth.get_config("tiny_peaked", dtype="bf16", batch=b, V=V, gamma=gamma, M=M, K2=K2, B=B,
                           approx="linear")
    _, reps = check(cfg)
    print(reps)


def test_bf16_linear_approximator_cluster_split_k():
    # 241 rows (two M-tiles), d = 512: K = 2d = 1024 split over the 4 CTAs of each cluster
    cfg = synth.get_config("tiny_peaked", dtype="bf16", batch=1, d=512, V=3000, gamma=16, M=16, K2=16,
                           B=32, approx="linear")
    check(cfg)


def test_bf16_zero_linear_approximator_equals_mary_marginal_tree():
    cfg = synth.get_config("tiny_peaked", dtype="bf16", batch=4, V=2000, approx="linear")
    inp = synth.make_inputs(cfg)
    inp["w_lin"].zero_()
    d = parity.device_inputs(inp)
    a = parity.run_gpu(cfg, d)
    b = parity.run_gpu(cfg.replace(mode="marginal_mary"), d)
    for k in ("node_tok", "node_parent", "node_depth", "node_score", "mask", "pos_ids"):
        np.testing.assert_array_equal(a[k], b[k], err_msg=k)


# ------------------------------------------------------------------ "w/ 2-prev" approximator
# (Sec. 4 "Model Design", Table 3): x = [h~ ; e(prev) ; e(token before prev)], one stage-2 row
# per pair of M-ary candidates (1 + M + M^2 (gamma - 2) rows), the child list of a node chosen
# by its own and its parent's candidate index; root_tok is [b, 2] = (x_t, x_{t-1}).


def test_fp32_two_prev_approximator():
    _, reps = check(synth.get_config("tiny_peaked", approx="swiglu_2prev"))
    print(reps)


@pytest.mark.parametrize("b,V", [(2, 2000), (4, 2304), (8, 2049)])
def test_bf16_two_prev_approximator_small(b, V):
    # 74 / 148 / 296 stage-2 rows: one, two and three M-tiles
    cfg = synth.get_config("tiny_peaked", dtype="bf16", batch=b, V=V, approx="swiglu_2prev")
    _, reps = check(cfg)
    print(reps)


def test_bf16_two_prev_approximator_cluster_split_k():
    # gamma 4, M 8: 137 rows (two M-tiles), d = I = 512: gate/up with K = 3d and the down
    # projection both split K over 4-CTA clusters; the residual rows come from the gather
    cfg = synth.get_config("tiny_peaked", dtype="bf16", batch=1, d=512, I=512, V=3000, gamma=4, M=8, K2=16,
                           B=32, approx="swiglu_2prev")
    check(cfg)


def test_fp32_two_prev_shared_queue_builder():
    # B = 200 > 127: the builder with its queue in shared memory takes the two-token rule too
    cfg = synth.get_config("tiny_peaked", V=4096, M=8, K2=200, B=200, approx="swiglu_2prev")
    _, reps = check(cfg)
    print(reps)


# ------------------------------------------------------------------ full sizes (the measured shapes)

_cache = {}


def _inputs(name, batch=None):
    key = (name, batch)
    if key not in _cache:
        _cache.clear()
        cfg = synth.get_config(name) if batch is None else synth.get_config(name, batch=batch)
        _cache[key] = synth.make_inputs(cfg)
    return _cache[key]


def _sequence(inp, s):
    """Sequence s of a batch of inputs as a batch of one (weights shared)."""
    per_seq = ("hidden", "root_tok", "root_pos", "root_prev")
    return {k: (v[s:s + 1] if k in per_seq and v is not None else v) for k, v in inp.items()}


@pytest.mark.parametrize("name", ["q8_b64", "q8_b32"])
def test_full_size_bf16_contract_over_sequences(name):
    # The measured shapes (one sequence per call, the launch configuration bench.py times) on
    # 8 sequences: one set of weights, 8 seeded hidden-state draws and root tokens. Every
    # sequence passes the stage-wise checks and the end-to-end contract; the counts show how
    # much of each tree the node-score bound decides.
    n = 8
    cfg8 = synth.get_config(name, batch=n)
    inp = _inputs(name, batch=n)
    W = parity.oracle_weights(inp)
    cfg = cfg8.replace(batch=1)
    agg = {}
    for s in range(n):
        _, reps = check(cfg, inp=_sequence(inp, s), W=W)
        for k, v in reps["e2e"].items():
            agg[k] = max(agg.get(k, 0), v) if k.startswith("max") else agg.get(k, 0) + v
    print(name, agg)
    assert agg["excluded_trees"] < n
    # the structural comparison must not be vacuous on these distributions (17 % of the cuts of
    # q8_b64, 34 % of q8_b32's are decided at the node bound)
    assert agg["cuts_determined"] >= 0.1 * agg["cuts"], agg


@pytest.mark.parametrize("name", ["q8_b64_linear", "q8_b32_2prev"])
def test_full_size_qwen3_8b_shape_variants(name):
    cfg = synth.get_config(name)
    inp = _inputs(name)
    W = parity.oracle_weights(inp)
    gpu, reps = check(cfg, inp=inp, W=W)
    print(name, reps)
    # the tree reaches as deep as the bf16-emulating oracle's tree (with two previous tokens the
    # random approximator's favourites are rarely stage-1 candidates, so both stay shallow)
    orc_e = parity.run_oracle(cfg, inp, emulate_bf16=True, W=W)[0]
    assert gpu["node_depth"][0].max() == orc_e.tree.depth.max()


@pytest.mark.parametrize("name", ["q8_b512", "q8_m64"])
def test_full_size_large_budget_and_branching(name):
    # Fig. 5 / Fig. 6 regimes at the full Qwen3-8B shape: B = K2 = 512 (exact lists), M = 64
    # (961 stage-2 rows)
    _, reps = check(synth.get_config(name), inp=_inputs(name))
    print(name, reps)


def test_full_size_batch32_sampled_sequences():
    cfg = synth.get_config("batch32")
    _, reps = check(cfg, orc_seqs=[0, 17, 31], emulate_also=False)
    print("batch32", reps["e2e"])


@pytest.mark.parametrize("name", ["wide_peaked", "wide_flat"])
def test_full_size_wide_sampled_sequence(name):
    cfg = synth.get_config(name)
    _, reps = check(cfg, orc_seqs=[3], emulate_also=False)
    print(name, reps["e2e"])


# ------------------------------------------------------------------ large budgets and branching
# (Fig. 5: budgets up to 512; Fig. 6: M up to 64): K2 = B keeps the per-row lists exact, the
# merge returns up to 512 entries, the builder tests membership among up to 64 candidates and
# keeps its queue in shared memory beyond B = 127.


def test_fp32_large_budget_and_branching():
    cfg = synth.get_config("tiny_peaked", M=64, K2=256, B=256)
    _, reps = check(cfg)
    print(reps)


def test_bf16_large_budget():
    cfg = synth.get_config("tiny_peaked", dtype="bf16", d=256, V=4096, M=48, K2=512, B=512)
    _, reps = check(cfg)
    print(reps)


def test_fp32_budget_near_the_limit_with_truncated_lists():
    # B = 1000 (the shared-memory queue at 32 slots per lane) with K2 = 512 < B: the oracle
    # truncates every list to 512 entries too
    cfg = synth.get_config("tiny_peaked", V=4096, M=32, K2=512, B=1000)
    _, reps = check(cfg)
    print(reps)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_lmhead_top512_equals_topk_of_exact_logits(dtype):
    # the merge's exact top-k at k = 512 against torch.topk of the fp64 logits (ties have
    # probability zero for these continuous inputs)
    from paper_2606_03819_gb300 import binding as Bn
    V, d, rows, k = 8192, 256, 20, 512
    dims = Bn.Dims(batch=rows, d=d, V=V, I=64, gamma=1, M=4, K2=k, B=k, dtype=dtype, mode="marginal")
    g = torch.Generator().manual_seed(11)
    dt = dims.torch_dtype
    W = (torch.randn(V, d, generator=g) * 0.02).to(dt)
    x = (torch.randn(rows, d, generator=g) * 4.0).to(dt)
    ws = Bn.alloc_workspace(dims)
    ids = torch.empty(rows, k, dtype=torch.int32, device="cuda")
    lp = torch.empty(rows, k, dtype=torch.float32, device="cuda")
    Bn.tf_status_reset(ws)
    Bn.tf_lmhead_partials(dims, W.cuda(), x.cuda(), rows, ws)
    Bn.tf_lmhead_merge(dims, W.cuda(), x.cuda(), rows, k, ids, lp, ws)
    assert not (Bn.tf_status_read(ws) & ~16)
    z = x.double() @ W.double().T
    ref = torch.topk(z, k, dim=1)
    lse = torch.logsumexp(z, dim=1, keepdim=True)
    got = ids.cpu().long()
    # the id sets must agree exactly wherever the k-th and (k+1)-th logits are apart by more
    # than the arithmetic's error (bf16 inputs, fp32 accumulation)
    tol = 1e-4 if dtype == "f32" else 2e-3
    zs = torch.sort(z, dim=1, descending=True).values
    for r in range(rows):
        if zs[r, k - 1] - zs[r, k] > tol:
            assert set(got[r].tolist()) == set(ref.indices[r].tolist()), f"row {r}"
        np.testing.assert_allclose(lp[r].cpu().double().numpy(), (z[r, got[r]] - lse[r]).numpy(), atol=tol)
    assert (lp[:, :-1] >= lp[:, 1:]).all()


def test_kernel_launch_counter_counts_each_kernel():
    # tf_stage1_marginals is one LM-head pass and one merge: two kernels per call
    from paper_2606_03819_gb300 import binding as Bn
    cfg = synth.get_config("tiny_peaked", dtype="bf16", batch=2, V=2000)
    d = parity.device_inputs(synth.make_inputs(cfg))
    dims = Bn.Dims.from_config(cfg)
    ws = Bn.alloc_workspace(dims)
    ids = torch.empty(cfg.batch, cfg.gamma, dims.K1, dtype=torch.int32, device="cuda")
    lp = torch.empty(cfg.batch, cfg.gamma, dims.K1, dtype=torch.float32, device="cuda")
    n0 = Bn.tf_kernel_launches()
    for _ in range(3):
        Bn.tf_stage1_marginals(dims, d, d["hidden"], ids, lp, ws)
    torch.cuda.synchronize()
    assert Bn.tf_kernel_launches() - n0 == 6
