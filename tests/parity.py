"""GPU-vs-oracle parity checks (test infrastructure; used by tests/ and __graft_entry__.smoke()).

Both sides read the same seeded inputs from synth/. The oracle runs in float64 (optionally with
bf16 rounding at the points where the CUDA path stores bf16). Comparison rules:

* log-probabilities (stage-1 top-K1, stage-2 top-K2, node scores): every value the GPU reports
  for a token id must be within `tol_lp` of the oracle's exact log-probability of that id, and
  the GPU's sorted values must match the oracle's sorted top values rank by rank within
  `tol_lp` (so a swap of two near-equal entries is allowed, a wrong value is not). Node scores
  are sums of up to depth log-probabilities and get depth * tol_lp.
* ids: the top-M candidate set of every depth (which decides the M-ary tree) must equal the
  oracle's whenever the oracle's gap at rank M exceeds `tol_sel`; stage-2 rows are paired with
  oracle rows by (depth, previous token).
* tree: when the oracle's order margin exceeds `tol_sel` the token, parent and depth arrays
  must be bit-exact (same pop order); when only the set margin does, the trees must be equal
  as sets of token paths. Otherwise only validity is checked (prefix-closed, M-ary rule,
  scores = sums of the GPU's own child log-probs).
* mask / position ids: always bit-exact against the oracle's mask of the GPU's own tree, and
  against the oracle's tree when that was required to match.
"""
from __future__ import annotations

import numpy as np
import torch

import synth
from oracle import treeflash_oracle as O

TOLS = {
    # lp: stage-1 log-probs vs the plain fp64 oracle; lp2: stage-2 log-probs vs the plain oracle,
    # on top of the oracle's own emulated-minus-plain difference (the bf16 path rounds x,
    # SiLU(G)*U and h' to bf16 before the next GEMM); lp_emul: everything vs the oracle that
    # rounds at those points (the
    # remaining difference is fp32-vs-fp64 accumulation flipping a bf16 rounding, worth up to
    # |w| * ulp(h') per flipped element); sel: selection margin above which the tree structure
    # must match exactly (twice the per-log-prob tolerance).
    "f32": dict(lp=1e-4, lp2=1e-4, lp_emul=1e-4, sel=1e-3),
    "bf16": dict(lp=2e-2, lp2=2e-2, lp_emul=2e-2, sel=4e-2),
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


def compare(cfg, gpu, orc, tol_lp, tol_sel, check_structure=True, tol_lp2=None, orc_round=None,
            round_factor=1.0):
    """Assert parity of one batch; returns a small report dict.

    orc_round: the bf16-emulating oracle's results for the same sequences. When given, every
    stage-2 row may additionally deviate by the oracle's own emulated-minus-plain difference at
    the reported ids (|gpu - plain| <= |gpu - emulated| + |emulated - plain|)."""
    tol_lp2 = tol_lp if tol_lp2 is None else tol_lp2
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
            if orc_round is not None:
                ekey = {k: r for r, k in enumerate(conditioning_keys(cfg, root, orc_round[s].top_ids, rprev))}
            for r, key in enumerate(gkeys):
                orow = okey.get(key)
                if orow is None:
                    rep["rows_s2_skipped"] += 1
                    continue
                tol_row = tol_lp2
                if orc_round is not None:
                    erow = ekey.get(key)
                    if erow is None:
                        rep["rows_s2_skipped"] += 1
                        continue
                    ids = gpu["child_ids"][s, r]
                    tol_row = tol_lp2 + round_factor * float(
                        np.abs(orc_round[s].s2_logp[erow][ids] - o.s2_logp[orow][ids]).max())
                    rep["max_round_allowance"] = max(rep.get("max_round_allowance", 0.0), tol_row - tol_lp2)
                e = _check_row(gpu["child_ids"][s, r], gpu["child_logp"][s, r], o.s2_logp[orow], tol_row,
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
                lim = np.maximum(dep[present], 1) * max(tol_lp, tol_lp2)
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
E2E_ROUND_FACTOR = 2.0   # stage-2 allowance vs the plain oracle, in units of the emulating
                         # oracle's own deviation (two realizations of the same bf16 storage)
E2E_TREE_MARGIN = 0.25   # plain-oracle set margin above which the trees must coincide


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
        err = max(err, _check_row(gpu["child_ids"][s, rr], gpu["child_logp"][s, rr], lp[r], 2e-2,
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
    """bf16 path against the plain fp64 oracle: stage 1 within 2e-2; every stage-2 row within
    2e-2 plus E2E_ROUND_FACTOR times the emulating oracle's own deviation from the plain one on
    that row (the effect of storing x, SiLU(G)*U and h' in bf16); trees equal as sets where the
    plain oracle's set margin exceeds E2E_TREE_MARGIN."""
    rep = compare(cfg, gpu, orc, 2e-2, np.inf, check_structure=False, tol_lp2=2e-2,
                  orc_round=orc_emul if cfg.mode == "ar" else None, round_factor=E2E_ROUND_FACTOR)
    rep["e2e_set_trees"] = 0
    for s, o in enumerate(orc):
        set_m, _ = O.selection_margins(o, cfg.M, cfg.K2, cfg.B, cfg.mode)
        if set_m > E2E_TREE_MARGIN:
            assert _paths(gpu["node_tok"][s], gpu["node_parent"][s]) == set(O.tree_paths(o.tree)), \
                f"seq {s}: tree differs from the plain oracle's"
            rep["e2e_set_trees"] += 1
    return rep
