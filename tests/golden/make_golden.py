"""Write the oracle's tiny fp32 trees (seed 0) to tiny_f32_seed0.json, and those of the
ablations' approximators (the linear layer, two previous tokens) to tiny_variants_seed0.json.

Calls only oracle/ and synth/. Run from the repository root:
    python tests/golden/make_golden.py
"""
import json
import os
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

import synth  # noqa: E402
from oracle import treeflash_oracle as O  # noqa: E402


def main():
    out = {}
    for name in ("tiny_f32", "tiny_peaked"):
        cfg = synth.get_config(name)
        inp = synth.make_inputs(cfg)
        W = O.weights_f64(inp, synth.to_f64)
        H = synth.to_f64(inp["hidden"])[0]
        res = O.draft_sequence(H, int(inp["root_tok"][0]), int(inp["root_pos"][0]), W,
                               M=cfg.M, K2=cfg.K2, B=cfg.B, temperature=cfg.temperature,
                               eps=cfg.rms_eps, mode=cfg.mode)
        out[name] = dict(tok=res.tree.tok.tolist(), parent=res.tree.parent.tolist(),
                         depth=res.tree.depth.tolist(),
                         score=[float(x) for x in res.tree.score],
                         top_ids=res.top_ids.tolist())
    with open(os.path.join(HERE, "tiny_f32_seed0.json"), "w") as f:
        json.dump(out, f, indent=1)
    variants = {}
    for approx in VARIANTS:
        cfg = synth.get_config("tiny_peaked", approx=approx)
        inp = synth.make_inputs(cfg)
        W = O.weights_f64(inp, synth.to_f64)
        H = synth.to_f64(inp["hidden"])[0]
        prev = int(inp["root_prev"][0]) if "root_prev" in inp else None
        res = O.draft_sequence(H, int(inp["root_tok"][0]), int(inp["root_pos"][0]), W,
                               M=cfg.M, K2=cfg.K2, B=cfg.B, temperature=cfg.temperature,
                               eps=cfg.rms_eps, mode=cfg.mode, approx=approx, root_prev=prev)
        variants["tiny_peaked/" + approx] = dict(
            tok=res.tree.tok.tolist(), parent=res.tree.parent.tolist(), depth=res.tree.depth.tolist(),
            score=[float(x) for x in res.tree.score], top_ids=res.top_ids.tolist(),
            child_logp_row0=[float(x) for x in res.child_logp[0]])
    with open(os.path.join(HERE, "tiny_variants_seed0.json"), "w") as f:
        json.dump(variants, f, indent=1)


VARIANTS = ("linear", "swiglu_2prev")


if __name__ == "__main__":
    main()
