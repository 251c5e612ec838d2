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
