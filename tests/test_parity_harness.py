"""The GPU parity harness accepts the oracle's own outputs (rounded to the GPU's output types)
and rejects planted mistakes, so a passing GPU test means something. Runs on CPU."""
import numpy as np
import pytest

import synth
import parity
from oracle import treeflash_oracle as O


def fake_gpu(cfg, orc, root_pos):
    b, n = cfg.batch, cfg.B + 1
    g = dict(top_ids=np.stack([o.top_ids for o in orc]).astype(np.int32),
             top_logp=np.stack([o.top_logp for o in orc]).astype(np.float32),
             node_tok=np.stack([o.tree.tok for o in orc]).astype(np.int32),
             node_parent=np.stack([o.tree.parent for o in orc]).astype(np.int32),
             node_depth=np.stack([o.tree.depth for o in orc]).astype(np.int32),
             node_score=np.stack([o.tree.score for o in orc]).astype(np.float32),
             mask=np.stack([o.mask for o in orc]), pos_ids=np.stack([o.pos for o in orc]).astype(np.int32),
             root_pos=np.asarray(root_pos), flags=0)
    if cfg.mode == "ar":
        g["child_ids"] = np.stack([o.child_ids for o in orc]).astype(np.int32)
        g["child_logp"] = np.stack([o.child_logp for o in orc]).astype(np.float32)
    return g


@pytest.mark.parametrize("mode", ["ar", "marginal", "marginal_mary"])
def test_harness_accepts_the_oracle(mode):
    cfg = synth.get_config("tiny_peaked", batch=2, mode=mode)
    inp = synth.make_inputs(cfg)
    orc = parity.run_oracle(cfg, inp)
    g = fake_gpu(cfg, orc, inp["root_pos"].numpy())
    rep = parity.compare(cfg, g, orc, 1e-4, 1e-3)
    assert rep["exact_trees"] + rep["set_trees"] + rep["valid_only_trees"] == 2


def test_harness_rejects_planted_mistakes():
    cfg = synth.get_config("tiny_peaked", batch=1)
    inp = synth.make_inputs(cfg)
    orc = parity.run_oracle(cfg, inp)
    base = fake_gpu(cfg, orc, inp["root_pos"].numpy())
    plants = []
    g = {k: (v.copy() if isinstance(v, np.ndarray) else v) for k, v in base.items()}
    g["top_logp"][0, 1, 0] += 1e-3; plants.append(g)                    # a wrong log-prob
    g = {k: (v.copy() if isinstance(v, np.ndarray) else v) for k, v in base.items()}
    g["child_ids"][0, 0, [0, 1]] = g["child_ids"][0, 0, [1, 0]]; plants.append(g)  # swapped ids
    g = {k: (v.copy() if isinstance(v, np.ndarray) else v) for k, v in base.items()}
    g["node_parent"][0, -1] = 0; plants.append(g)                       # a rewired node
    g = {k: (v.copy() if isinstance(v, np.ndarray) else v) for k, v in base.items()}
    g["mask"][0, 3, 0] = 0; plants.append(g)                            # a broken mask
    for g in plants:
        with pytest.raises(AssertionError):
            parity.compare(cfg, g, orc, 1e-4, 1e-3)


@pytest.mark.parametrize("approx", ["linear", "swiglu_2prev"])
def test_harness_accepts_the_oracle_for_the_ablation_approximators(approx):
    cfg = synth.get_config("tiny_peaked", batch=2, approx=approx)
    inp = synth.make_inputs(cfg)
    orc = parity.run_oracle(cfg, inp)
    g = fake_gpu(cfg, orc, inp["root_pos"].numpy())
    if approx == "swiglu_2prev":
        g["root_prev"] = inp["root_prev"].numpy()
        assert g["child_ids"].shape[1] == cfg.R == 37
    rep = parity.compare(cfg, g, orc, 1e-4, 1e-3)
    assert rep["rows_s2"] == 2 * cfg.R and rep["rows_s2_skipped"] == 0


def test_harness_rejects_two_prev_rows_swapped_within_a_depth():
    # rows (depth 3, m1 = 0, m2 = 0) and (depth 3, m1 = 0, m2 = 1) share the previous token and
    # differ only in the token before it: pairing rows by the previous token alone would miss
    # the swap
    cfg = synth.get_config("tiny_peaked", batch=1, approx="swiglu_2prev", wd_std=2.0)
    inp = synth.make_inputs(cfg)
    orc = parity.run_oracle(cfg, inp)
    g = fake_gpu(cfg, orc, inp["root_pos"].numpy())
    g["root_prev"] = inp["root_prev"].numpy()
    r = 1 + cfg.M
    assert np.abs(orc[0].child_logp[r] - orc[0].child_logp[r + 1]).max() > 1e-3
    for k in ("child_ids", "child_logp"):
        g[k][0, [r, r + 1]] = g[k][0, [r + 1, r]]
    with pytest.raises(AssertionError):
        parity.compare(cfg, g, orc, 1e-4, 1e-3, check_structure=False)


# ------------------------------------------------------------------ the bf16 end-to-end contract


def _bf16_case(B=16, seed=0):
    cfg = synth.get_config("tiny_peaked", batch=2, K2=B, B=B)
    inp = synth.make_inputs(cfg, seed=seed)
    orc = parity.run_oracle(cfg, inp)
    orc_e = parity.run_oracle(cfg, inp, emulate_bf16=True)
    return cfg, inp, orc, orc_e


def test_bf16_contract_accepts_the_emulating_oracle():
    # the emulating oracle's own outputs pass, with every cut decided (its scores are exact
    # against itself) and the whole tree compared bit for bit
    cfg, inp, orc, orc_e = _bf16_case()
    g = fake_gpu(cfg, orc_e, inp["root_pos"].numpy())
    rep = parity.check_bf16_end_to_end(cfg, g, orc, orc_e)
    assert rep["excluded_trees"] == 0 and rep["rows_s2"] == 2 * cfg.R
    assert rep["cuts"] == 2 * cfg.B and rep["cuts_determined"] > 0
    assert rep["exact_trees"] + rep["set_trees"] <= 2
    assert rep["max_err_node"] < 1e-5


def test_bf16_contract_rejects_a_swapped_node_at_a_decided_cut():
    # replace the last node of a tree by the best node left out: wherever the cut at B is
    # decided, the contract must notice
    cfg, inp, orc, orc_e = _bf16_case()
    base = fake_gpu(cfg, orc_e, inp["root_pos"].numpy())
    hit = 0
    for s in range(cfg.batch):
        e = orc_e[s]
        src = O.ChildSource(cfg.mode, cfg.gamma, cfg.M, e.top_ids, e.s1_logp, e.s2_logp)
        big = O.build_tree_lazy(src, int(e.tree.tok[0]), cfg.B + 1)
        pops = [p[0] for p in big.pops]
        if pops[cfg.B - 1] - pops[cfg.B] <= 2 * parity.BF16["node"]:
            continue          # the cut at B is not decided: nothing to assert there
        if big.parent[cfg.B + 1] == cfg.B:
            continue          # the left-out node hangs below the node it would replace
        g = {k: (v.copy() if isinstance(v, np.ndarray) else v) for k, v in base.items()}
        for k, src_arr in (("node_tok", big.tok), ("node_parent", big.parent), ("node_depth", big.depth)):
            g[k][s, cfg.B] = src_arr[cfg.B + 1]
        g["node_score"][s, cfg.B] = pops[cfg.B]
        m, pos = O.tree_mask(g["node_parent"][s].astype(np.int64), g["node_depth"][s].astype(np.int64),
                             int(g["root_pos"][s]))
        g["mask"][s], g["pos_ids"][s] = m, pos
        with pytest.raises(AssertionError):
            parity.check_bf16_end_to_end(cfg, g, orc, orc_e)
        hit += 1
    assert hit > 0, "no sequence with a decided cut at B to plant the mistake in"


def test_bf16_contract_rejects_stage2_values_beyond_the_bound():
    cfg, inp, orc, orc_e = _bf16_case()
    g = fake_gpu(cfg, orc_e, inp["root_pos"].numpy())
    g["child_logp"][0, 3, 0] += 1.5 * parity.BF16["s2"]
    with pytest.raises(AssertionError):
        parity.check_bf16_end_to_end(cfg, g, orc, orc_e)
