"""GPU-vs-oracle parity checks (test infrastructure; used by tests/ and __graft_entry__.smoke()).

Both sides read the same seeded inputs from synth/. The oracle runs in float64 (optionally with
bf16 rounding at the points where the CUDA path stores bf16). Comparison rules:

* log-probabilities (stage-1 top-K1, stage-2 top-K2, node scores): every value the GPU reports
  for a token id must be within the bound of the oracle's exact log-probability of that id, and
  the GPU's sorted values must match the oracle's sorted top values rank by rank (so a swap of
  two near-equal entries is allowed, a wrong value is not); stage-2 rows are paired with oracle
  rows by their conditioning (depth, previous token(s)).
* fp32 path (compare): everything against the plain oracle within 1e-4; the top-M candidate
  sets, and the tree's tokens, parents, depths, mask and position ids, bit-exact wherever the
  oracle's selection margins exceed 1e-3 (as sets of token paths where only the set margin does).
* bf16 path (check_bf16_end_to_end, BF16): stage 1 against the plain oracle, stage 2 and the
  tree against the oracle that rounds to bf16 where the GPU stores bf16; the structure is
  compared at every cut of the oracle's pop order that the node-score bound decides. Each stage
  is also checked on the GPU's own inputs to it (check_bf16_stagewise).
* mask / position ids: always bit-exact against the oracle's mask of the GPU's own tree.
"""
from __future__ import annotations

import numpy as np
import torch

import synth
from oracle import treeflash_oracle as O

TOLS = {
    # fp32 path against the plain fp64 oracle: lp, every log-probability; sel, the selection
    # margin above which the tree structure must match exactly. The bf16 path's bounds are BF16.
    "f32": dict(lp=1e-4, sel=1e-3),
}


def oracle_weights(inp):
    return O.weights_f64(inp, synth.to_f64)


def run_oracle(cfg, inp, emulate_bf16=False, seqs=None, W=None):
    W = W if W is not None else oracle_weights(inp)
    H = synth.to_f64(inp["hidden"])
    seqs = range(cfg.batch) if seqs is None else seqs
    out = []
    for s in seqs:
        prev = int(inp["root_prev"][s]) if inp.get("root_prev") is not None else None
        out.append(O.draft_sequence(H[s], int(inp["root_tok"][s]), int(inp["root_pos"][s]), W,
                                    M=cfg.M, K2=cfg.K2, B=cfg.B, temperature=cfg.temperature,
                                    eps=cfg.rms_eps, mode=cfg.mode, emulate_bf16=emulate_bf16,
                                    keep=cfg.K2 if cfg.K2 < cfg.B else None, approx=cfg.approx,
                                    root_prev=prev))
    return out


def device_inputs(inp, device="cuda"):
    """The GPU's inputs. With a token before each root (the two-previous-token approximator)
    root_tok becomes the [b, 2] array (x_t, x_{t-1}) the C ABI takes in that mode."""
    keys = ("hidden", "lm_head", "embed", "norm_h", "norm_e", "w_gate", "w_up", "w_down", "w_lin",
            "root_tok", "root_pos")
    out = {k: inp[k].to(device).contiguous() for k in keys if inp.get(k) is not None}
    if inp.get("root_prev") is not None:
        out["root_tok"] = torch.stack([inp["root_tok"], inp["root_prev"]], dim=1).to(device).contiguous()
    return out


def conditioning_keys(cfg, root_tok, top_ids, root_prev=None):
    """Per stage-2 row, the key that identifies its conditioning: (depth index, previous token)
    or, with two previous tokens, (depth index, previous token, the token before it)."""
    if cfg.approx == "swiglu_2prev":
        hid, p1, p2 = O.stage2_conditioning_2prev(cfg.gamma, cfg.M, root_tok, root_prev, top_ids)
        return [(int(h), int(a), int(b)) for h, a, b in zip(hid, p1, p2)]
    hid, prev = O.stage2_conditioning(cfg.gamma, cfg.M, root_tok, top_ids)
    return [(int(h), int(p)) for h, p in zip(hid, prev)]


def stage2_row_of(cfg, top_ids_s, tok, par, dep, i):
    """Index of the stage-2 row node i's token was drawn from (TreeFlash mode), by the M-ary
    candidate indices of its ancestors; asserts that its parent (and, with two previous tokens,
    its grandparent) lies in the M-ary tree."""
    M = cfg.M
    if dep[i] == 1:
        return 0
    p = int(par[i])
    cand = top_ids_s[dep[p] - 1, :M].tolist()
    assert int(tok[p]) in cand, f"node {p} expanded outside the M-ary tree"
    m = cand.index(int(tok[p]))
    if cfg.approx != "swiglu_2prev":
        return 1 + (dep[p] - 1) * M + m
    if dep[p] == 1:
        return 1 + m
    gp = int(par[p])
    gcand = top_ids_s[dep[gp] - 1, :M].tolist()
    assert int(tok[gp]) in gcand, f"node {gp} expanded outside the M-ary tree"
    return 1 + M + (dep[p] - 2) * M * M + m * M + gcand.index(int(tok[gp]))


def run_gpu(cfg, dinp, drafter=None):
    from paper_2606_03819_gb300 import Dims, Drafter
    dims = Dims.from_config(cfg)
    dr = drafter or Drafter(dims, dinp)
    out = dr.draft(dinp["hidden"], dinp["root_tok"], dinp["root_pos"])
    flags = dr.status()
    res = {k: (v.cpu().numpy() if v is not None else None) for k, v in out.items()}
    res["flags"] = flags
    res["root_pos"] = dinp["root_pos"].cpu().numpy()
    if dinp["root_tok"].dim() == 2:        # (x_t, x_{t-1}) per sequence
        res["root_prev"] = dinp["root_tok"][:, 1].cpu().numpy()
    if cfg.mode == "ar":
        from paper_2606_03819_gb300 import binding as Bn
        views = (("X", Bn.TF_VIEW_X), ("A", Bn.TF_VIEW_A), ("hp", Bn.TF_VIEW_H_PRIME))
        for name, view in views:
            if name == "A" and cfg.approx == "linear":   # no SwiGLU intermediate
                continue
            res[name] = Bn.tf_workspace_view(dims, dr.ws, view).double().cpu().numpy()
    return res


def _check_row(gpu_ids, gpu_lp, full_lp, tol, what):
    """GPU top list vs the oracle's full distribution of the same row."""
    ids = np.asarray(gpu_ids)
    assert (ids >= 0).all() and (ids < full_lp.shape[0]).all(), f"{what}: id out of range"
    assert len(set(ids.tolist())) == len(ids), f"{what}: duplicate ids"
    err_id = np.abs(gpu_lp - full_lp[ids]).max()
    top = np.sort(full_lp)[::-1][: len(ids)]
    err_rank = np.abs(np.sort(gpu_lp)[::-1] - top).max()
    assert err_id <= tol, f"{what}: logp of reported ids off by {err_id:.3g} > {tol}"
    assert err_rank <= tol, f"{what}: sorted top values off by {err_rank:.3g} > {tol}"
    return max(err_id, err_rank)


def compare(cfg, gpu, orc, tol_lp, tol_sel, check_structure=True):
    """Assert parity of one batch against one oracle result per sequence (the fp32 path's
    rule: every log-probability within tol_lp, structure exact beyond tol_sel); returns a small
    report dict."""
    rep = dict(max_err_s1=0.0, max_err_s2=0.0, max_err_score=0.0, rows_s2=0, rows_s2_skipped=0,
               exact_trees=0, set_trees=0, valid_only_trees=0)
    M, g = cfg.M, cfg.gamma
    for s, o in enumerate(orc):
        # ---- stage 1
        for i in range(g):
            e = _check_row(gpu["top_ids"][s, i], gpu["top_logp"][s, i], o.s1_logp[i], tol_lp, f"seq {s} depth {i + 1}")
            rep["max_err_s1"] = max(rep["max_err_s1"], e)
            if i < g - 1 and O.topk_margin(o.s1_logp[i], M) > tol_sel:
                assert set(gpu["top_ids"][s, i, :M].tolist()) == set(o.top_ids[i, :M].tolist()), \
                    f"seq {s} depth {i + 1}: top-M set differs"
        # ---- stage 2, rows paired by (depth, previous token(s))
        if cfg.mode == "ar":
            root = int(o.tree.tok[0])
            rprev = int(gpu["root_prev"][s]) if gpu.get("root_prev") is not None else None
            okey = {k: r for r, k in enumerate(conditioning_keys(cfg, root, o.top_ids, rprev))}
            gkeys = conditioning_keys(cfg, root, gpu["top_ids"][s], rprev)
            for r, key in enumerate(gkeys):
                orow = okey.get(key)
                if orow is None:
                    rep["rows_s2_skipped"] += 1
                    continue
                e = _check_row(gpu["child_ids"][s, r], gpu["child_logp"][s, r], o.s2_logp[orow], tol_lp,
                               f"seq {s} stage-2 row {r}")
                rep["max_err_s2"] = max(rep["max_err_s2"], e)
                rep["rows_s2"] += 1
        # ---- tree
        tok, par, dep, sc = (gpu["node_tok"][s], gpu["node_parent"][s], gpu["node_depth"][s],
                             gpu["node_score"][s])
        _check_tree_valid(cfg, gpu, s)
        if check_structure:
            set_m, order_m = O.selection_margins(o, M, cfg.K2, cfg.B, cfg.mode)
            if order_m > tol_sel:
                np.testing.assert_array_equal(tok, o.tree.tok, err_msg=f"seq {s} tokens")
                np.testing.assert_array_equal(par, o.tree.parent, err_msg=f"seq {s} parents")
                np.testing.assert_array_equal(dep, o.tree.depth, err_msg=f"seq {s} depths")
                np.testing.assert_array_equal(gpu["mask"][s], o.mask, err_msg=f"seq {s} mask")
                np.testing.assert_array_equal(gpu["pos_ids"][s], o.pos, err_msg=f"seq {s} pos")
                present = o.tree.parent >= 0
                present[0] = True
                err = np.abs(sc[present] - o.tree.score[present])
                lim = np.maximum(dep[present], 1) * tol_lp
                assert (err <= lim).all(), f"seq {s}: node score off by {err.max():.3g}"
                rep["max_err_score"] = max(rep["max_err_score"], float(err.max()))
                rep["exact_trees"] += 1
            elif set_m > tol_sel:
                gp = _paths(tok, par)
                assert gp == set(O.tree_paths(o.tree)), f"seq {s}: tree differs as a set"
                rep["set_trees"] += 1
            else:
                rep["valid_only_trees"] += 1
        # ---- mask of the GPU's own tree
        m, pos = O.tree_mask(par.astype(np.int64), dep.astype(np.int64), int(gpu["root_pos"][s]))
        np.testing.assert_array_equal(gpu["mask"][s], m, err_msg=f"seq {s} mask of own tree")
        np.testing.assert_array_equal(gpu["pos_ids"][s], pos, err_msg=f"seq {s} pos of own tree")
    return rep


def _paths(tok, par):
    paths = {0: ()}
    out = set()
    for i in range(1, tok.shape[0]):
        if par[i] < 0:
            continue
        paths[i] = paths[int(par[i])] + (int(tok[i]),)
        out.add(paths[i])
    return out


def _check_tree_valid(cfg, gpu, s):
    tok, par, dep, sc = (gpu["node_tok"][s], gpu["node_parent"][s], gpu["node_depth"][s], gpu["node_score"][s])
    n = cfg.B + 1
    assert tok.shape == (n,)
    assert par[0] == -1 and dep[0] == 0 and sc[0] == 0.0
    seen = set()
    for i in range(1, n):
        p = int(par[i])
        if p < 0:
            assert tok[i] == -1 and dep[i] == -1
            continue
        assert 0 <= p < i, f"seq {s} node {i}: parent {p}"
        assert dep[i] == dep[p] + 1 <= cfg.gamma
        assert sc[i] <= sc[p] + 1e-6
        assert (p, int(tok[i])) not in seen
        seen.add((p, int(tok[i])))
        # score = parent score + the GPU's own log-prob of this token in the child list used
        if cfg.mode == "ar":
            row = stage2_row_of(cfg, gpu["top_ids"][s], tok, par, dep, i)
            ids, lp = gpu["child_ids"][s, row], gpu["child_logp"][s, row]
        else:
            if cfg.mode == "marginal_mary" and dep[i] > 1:
                assert int(tok[p]) in gpu["top_ids"][s, dep[p] - 1, : cfg.M].tolist()
            ids, lp = gpu["top_ids"][s, dep[i] - 1, : cfg.K2], gpu["top_logp"][s, dep[i] - 1, : cfg.K2]
        where = np.nonzero(ids == tok[i])[0]
        assert where.size == 1, f"seq {s} node {i}: token not in its child list"
        assert abs(sc[i] - (sc[p] + lp[where[0]])) <= 1e-5 * max(1.0, abs(sc[i]))


# ------------------------------------------------------------------------------------------
# bf16 path: stage-by-stage parity. Storing x, SiLU(G)*U and h' in bf16 makes the end-to-end
# result sensitive at the ulp level (one element rounded the other way perturbs every later dot
# product), so each kernel is checked against the oracle's formula applied to the GPU's own
# inputs of that stage, with the error allowed by bf16 rounding and fp32 accumulation; the end
# to end result is then checked against the plain fp64 oracle with a bound for that storage.
# ------------------------------------------------------------------------------------------

ACC_REL = 2.0 ** -14     # tensor-core fp32 accumulation: relative to the sum of |terms|

# The bf16 end-to-end contract. The paper runs its method in bf16 (Sec. 4, Setup), and this path
# stores x, SiLU(G)*U and h' in bf16 between its tensor-core GEMMs (reading R11). The reference
# is therefore the oracle that rounds at exactly those points; what remains between the two is
# fp32 tensor-core accumulation against fp64, which flips a small fraction of those roundings.
#  s1:   stage-1 log-probabilities against the plain oracle (bf16 inputs, nothing rounded before
#        them, fp32 accumulation): measured at most 1.5e-4 over the full-size workloads.
#  s2:   stage-2 log-probabilities against the emulating oracle, every reported id and rank by
#        rank. Measured maxima on the full-size workloads: q8_b32 0.024 and q8_b64 0.031 (8
#        sequences each, 247k entries; median 0.0012), q8_b512 0.025, q8_m64 0.033, batch32
#        0.025, q8_b32_2prev 0.048, wide_flat 0.040, wide_peaked 0.054 (its larger hidden states
#        make each flipped bf16 rounding of h' weigh more). The bound is about twice the largest.
#        Against the plain oracle the same entries differ by up to 0.14, as much as the
#        emulating oracle itself differs from the plain one: the bf16 storage, not the kernels.
#  node: node scores (sums of log-probabilities along a path) against the emulating oracle's
#        score of the same path: measured at most 0.028 (wide_peaked; batch32 0.027, q8_b64
#        0.0155 over 8 trees), with no growth in depth (the tree uses each row's best entries,
#        where the log-sum-exp error cancels). The bound is about twice the largest; it decides
#        where the structure must match.
BF16 = dict(s1=1e-3, s2=0.1, node=0.06)
UNIVERSE_EXTRA = 16      # universe nodes listed beyond the budget for the cut test


def _ulp_bf16(x):
    x = np.abs(np.asarray(x, dtype=np.float64))
    return np.ldexp(1.0, np.frexp(np.maximum(x, 1e-30))[1] - 8)


def check_bf16_stagewise(cfg, inp, W, gpu):
    """Per-stage parity of the bf16 tensor-core path for every sequence; returns a report."""
    rep = {}
    g, M, d, I, R = cfg.gamma, cfg.M, cfg.d, cfg.I, cfg.R
    H = synth.to_f64(inp["hidden"])
    rows_h, rows_prev, rows_prev2 = [], [], []
    for s in range(cfg.batch):
        if cfg.approx == "swiglu_2prev":
            hid, prev, prev2 = O.stage2_conditioning_2prev(g, M, int(inp["root_tok"][s]), int(inp["root_prev"][s]),
                                                           gpu["top_ids"][s])
            rows_prev2.append(prev2)
        else:
            hid, prev = O.stage2_conditioning(g, M, int(inp["root_tok"][s]), gpu["top_ids"][s])
        rows_h.append(H[s][hid])
        rows_prev.append(prev)
    Hr = np.concatenate(rows_h)
    prev = np.concatenate(rows_prev)
    # x: correctly rounded normalisations (computed without per-element fp64 on the GPU)
    parts = [O.bf16_round(O.rmsnorm(Hr, W["norm_h"], cfg.rms_eps)),
             O.bf16_round(O.rmsnorm(W["embed"][prev], W["norm_e"], cfg.rms_eps))]
    if rows_prev2:
        parts.append(O.bf16_round(O.rmsnorm(W["embed"][np.concatenate(rows_prev2)], W["norm_e"], cfg.rms_eps)))
    x_ref = np.concatenate(parts, axis=1)
    X = gpu["X"]
    rep["x_mismatch_frac"] = float((X != x_ref).mean())
    assert np.all(np.abs(X - x_ref) <= _ulp_bf16(x_ref)), "x off by more than one bf16 ulp"
    assert rep["x_mismatch_frac"] < 1e-4
    if cfg.approx == "linear":
        # h' = h + W_lin x from the GPU's x: one GEMM, one bf16 rounding of the fp32 sum
        SD = np.abs(X) @ np.abs(W["w_lin"]).T
        hp_exact = Hr + X @ W["w_lin"].T
    else:
        SD, hp_exact = _swiglu_stage(W, X, gpu, rep, Hr)
    hp = gpu["hp"]
    rep["hp_round_flip_frac"] = float((hp != O.bf16_round(hp_exact)).mean())
    assert np.all(np.abs(hp - hp_exact) <= _ulp_bf16(hp_exact) + ACC_REL * SD), "h' off"
    _check_lmhead_and_builder(cfg, W, gpu, hp, rep)
    return rep


def _swiglu_stage(W, X, gpu, rep, Hr):
    """SiLU(G)*U of the GPU's x within one bf16 ulp plus the accumulation bound; returns the
    bound's sum of |terms| and the exact h' of the GPU's A."""
    # A from the GPU's x
    G, U = X @ W["w_gate"].T, X @ W["w_up"].T
    SG, SU = np.abs(X) @ np.abs(W["w_gate"]).T, np.abs(X) @ np.abs(W["w_up"]).T
    a_exact = O.silu(G) * U
    sig = 1.0 / (1.0 + np.exp(-G))
    dsilu = sig * (1 + G * (1 - sig))
    a_tol = _ulp_bf16(a_exact) + ACC_REL * (np.abs(dsilu * U) * SG + np.abs(O.silu(G)) * SU)
    A = gpu["A"]
    rep["A_round_flip_frac"] = float((A != O.bf16_round(a_exact)).mean())
    assert np.all(np.abs(A - a_exact) <= a_tol), "SiLU(G)*U off by more than rounding + accumulation"
    # h' from the GPU's A
    return np.abs(A) @ np.abs(W["w_down"]).T, Hr + A @ W["w_down"].T


def _check_lmhead_and_builder(cfg, W, gpu, hp, rep):
    R = cfg.R
    # LM head + log-softmax + top-k of the GPU's own h'
    lp = O.log_softmax(O.lm_head(hp, W["lm_head"], cfg.temperature))
    err = 0.0
    for r in range(hp.shape[0]):
        s, rr = divmod(r, R)
        err = max(err, _check_row(gpu["child_ids"][s, rr], gpu["child_logp"][s, rr], lp[r], BF16["s1"],
                                  f"seq {s} stage-2 row {rr} (LM head of the GPU's h')"))
    rep["lmhead_logp_err"] = err
    # Part 2 on the GPU's own lists: the oracle's builder must pick the same tree
    rep["builder_exact"] = rep["builder_set"] = 0
    for s in range(cfg.batch):
        src = _gpu_lists_source(cfg, gpu, s)
        t = O.build_tree_lazy(src, int(gpu["node_tok"][s, 0]), cfg.B, keep=cfg.K2)
        scores = [p[0] for p in t.pops]
        adj = min([a - b for a, b in zip(scores, scores[1:])] + [np.inf])
        if adj > 1e-5:
            np.testing.assert_array_equal(gpu["node_tok"][s], t.tok, err_msg=f"seq {s} builder tokens")
            np.testing.assert_array_equal(gpu["node_parent"][s], t.parent, err_msg=f"seq {s} builder parents")
            np.testing.assert_allclose(gpu["node_score"][s][t.parent >= 0], t.score[t.parent >= 0], atol=1e-4)
            rep["builder_exact"] += 1
        else:
            assert _paths(gpu["node_tok"][s], gpu["node_parent"][s]) == set(O.tree_paths(t))
            rep["builder_set"] += 1
    return rep


def _gpu_lists_source(cfg, gpu, s):
    """An oracle ChildSource whose distributions are the GPU's own top-k lists (other entries
    -inf), so the oracle's Part 2 runs on exactly the GPU's inputs."""
    V = cfg.V

    def dense(ids, lp):
        row = np.full(V, -np.inf)
        row[ids] = lp.astype(np.float64)
        return row
    s1 = np.stack([dense(gpu["top_ids"][s, i], gpu["top_logp"][s, i]) for i in range(cfg.gamma)])
    s2 = None
    if cfg.mode == "ar":
        s2 = np.stack([dense(gpu["child_ids"][s, r], gpu["child_logp"][s, r]) for r in range(cfg.R)])
    return O.ChildSource(cfg.mode, cfg.gamma, cfg.M, gpu["top_ids"][s].astype(np.int64), s1, s2, cfg.approx)


def check_bf16_end_to_end(cfg, gpu, orc, orc_emul):
    """The bf16 path end to end (BF16 explains the bounds). orc: the plain fp64 oracle;
    orc_emul: the oracle that rounds x, SiLU(G)*U and h' to bf16 where the GPU stores them (None
    in the marginal modes, where nothing is stored in bf16 before the log-probabilities)."""
    T = BF16
    ar = cfg.mode == "ar"
    ref = orc_emul if ar else orc
    M, g = cfg.M, cfg.gamma
    rep = dict(max_err_s1=0.0, max_err_s2_emul=0.0, max_err_s2_plain=0.0, max_emul_minus_plain=0.0,
               max_err_node=0.0, rows_s2=0, rows_s2_skipped=0, cuts=0, cuts_determined=0,
               prefix_nodes=0, exact_trees=0, set_trees=0, excluded_trees=0)
    for s, (o, e) in enumerate(zip(orc, ref)):
        # ---- stage 1 against the plain oracle (nothing is rounded before it)
        for i in range(g):
            err = _check_row(gpu["top_ids"][s, i], gpu["top_logp"][s, i], o.s1_logp[i], T["s1"],
                             f"seq {s} depth {i + 1}")
            rep["max_err_s1"] = max(rep["max_err_s1"], err)
        # the M-ary candidate sets decide the tree's universe: equal wherever the gap at rank M
        # exceeds twice the stage-1 bound; a set inside that band excludes the tree below
        same_sets = True
        if cfg.mode != "marginal":
            for i in range(g - 1):
                if set(gpu["top_ids"][s, i, :M].tolist()) != set(o.top_ids[i, :M].tolist()):
                    assert O.topk_margin(o.s1_logp[i], M) <= 2 * T["s1"], f"seq {s} depth {i + 1}: top-M set differs"
                    same_sets = False
        # ---- stage 2 against the emulating oracle, rows paired by their conditioning
        if ar:
            root = int(o.tree.tok[0])
            rprev = int(gpu["root_prev"][s]) if gpu.get("root_prev") is not None else None
            ekey = {k: r for r, k in enumerate(conditioning_keys(cfg, root, e.top_ids, rprev))}
            for r, key in enumerate(conditioning_keys(cfg, root, gpu["top_ids"][s], rprev)):
                erow = ekey.get(key)
                if erow is None:
                    rep["rows_s2_skipped"] += 1
                    continue
                ids, lp = gpu["child_ids"][s, r], gpu["child_logp"][s, r]
                err = _check_row(ids, lp, e.s2_logp[erow], T["s2"], f"seq {s} stage-2 row {r}")
                rep["max_err_s2_emul"] = max(rep["max_err_s2_emul"], err)
                # reported, not bounded: the plain oracle stores nothing in bf16
                rep["max_err_s2_plain"] = max(rep["max_err_s2_plain"], float(np.abs(lp - o.s2_logp[erow][ids]).max()))
                rep["max_emul_minus_plain"] = max(rep["max_emul_minus_plain"],
                                                  float(np.abs(e.s2_logp[erow][ids] - o.s2_logp[erow][ids]).max()))
                rep["rows_s2"] += 1
        # ---- tree: valid, its mask exact, and its structure against the reference oracle's
        _check_tree_valid(cfg, gpu, s)
        par, dep = gpu["node_parent"][s], gpu["node_depth"][s]
        m, pos = O.tree_mask(par.astype(np.int64), dep.astype(np.int64), int(gpu["root_pos"][s]))
        np.testing.assert_array_equal(gpu["mask"][s], m, err_msg=f"seq {s} mask of own tree")
        np.testing.assert_array_equal(gpu["pos_ids"][s], pos, err_msg=f"seq {s} pos of own tree")
        if not same_sets:
            rep["excluded_trees"] += 1
            continue
        tau = T["node"] if ar else g * T["s1"]
        _compare_cuts(cfg, gpu, s, e, tau, rep)
    return rep


def _compare_cuts(cfg, gpu, s, e, tau, rep):
    """Structure of the GPU's tree against the oracle result e wherever tau decides it.

    The oracle's universe in pop order (the B best nodes and UNIVERSE_EXTRA more) has scores
    s_1 >= s_2 >= ...; every GPU node score is within tau of the oracle's score of the same
    path. The set of the j best nodes is then the same on both sides whenever
    min over i <= j of (s_i - tau) > max over i > j of (s_i + tau) (nodes beyond the listed
    ones score at most the last listed score). At every such cut j the GPU's first j nodes must
    be the oracle's first j nodes as a set of token paths; over the longest run of such cuts from
    j = 1 the pop order is fixed, so tokens, parents and depths must match bit for bit; with every
    cut up to B decided the whole tree, its mask and position ids must."""
    B = cfg.B
    src = O.ChildSource(cfg.mode, cfg.gamma, cfg.M, e.top_ids, e.s1_logp, e.s2_logp, cfg.approx)
    root = int(e.tree.tok[0])
    keep = cfg.K2 if cfg.K2 < B else None
    big = O.build_tree_lazy(src, root, B + UNIVERSE_EXTRA, keep)
    pops = np.array([p[0] for p in big.pops], dtype=np.float64)
    ep = O.tree_paths(big)
    n = len(pops)
    gp = []
    paths = {0: ()}
    for i in range(1, B + 1):
        if gpu["node_parent"][s, i] < 0:
            gp.append(None)
            continue
        paths[i] = paths[int(gpu["node_parent"][s, i])] + (int(gpu["node_tok"][s, i]),)
        gp.append(paths[i])
    # GPU node scores against the oracle's scores of the same paths
    es = dict(zip(ep, pops))
    for i, p in enumerate(gp):
        if p is not None and p in es:
            err = abs(float(gpu["node_score"][s, i + 1]) - es[p])
            assert err <= tau, f"seq {s} node {i + 1}: score off by {err:.3g} > {tau}"
            rep["max_err_node"] = max(rep["max_err_node"], err)
    lo = np.minimum.accumulate(pops - tau)
    hi = np.maximum.accumulate((pops + tau)[::-1])[::-1]
    tail = pops[-1] + tau if n == B + UNIVERSE_EXTRA else -np.inf   # else the universe is exhausted
    decided = []
    for j in range(1, min(B, n) + 1):
        outside = max(hi[j] if j < n else -np.inf, tail)
        if lo[j - 1] > outside:
            decided.append(j)
            assert set(gp[:j]) == set(ep[:j]), f"seq {s}: the best {j} nodes differ from the oracle's"
    rep["cuts"] += B
    rep["cuts_determined"] += len(decided)
    prefix = 0
    while prefix < len(decided) and decided[prefix] == prefix + 1:
        prefix += 1
    ref_tok, ref_par, ref_dep = big.tok[: B + 1], big.parent[: B + 1], big.depth[: B + 1]
    np.testing.assert_array_equal(gpu["node_tok"][s, : prefix + 1], ref_tok[: prefix + 1], err_msg=f"seq {s} tokens")
    np.testing.assert_array_equal(gpu["node_parent"][s, : prefix + 1], ref_par[: prefix + 1], err_msg=f"seq {s} parents")
    np.testing.assert_array_equal(gpu["node_depth"][s, : prefix + 1], ref_dep[: prefix + 1], err_msg=f"seq {s} depths")
    rep["prefix_nodes"] += prefix
    if prefix == B and n >= B:
        m, pos = O.tree_mask(ref_par.astype(np.int64), ref_dep.astype(np.int64), int(gpu["root_pos"][s]))
        np.testing.assert_array_equal(gpu["mask"][s], m, err_msg=f"seq {s} mask")
        np.testing.assert_array_equal(gpu["pos_ids"][s], pos, err_msg=f"seq {s} pos")
        rep["exact_trees"] += 1
    elif B in decided:
        rep["set_trees"] += 1
