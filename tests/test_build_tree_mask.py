"""tf_build_tree_mask against tf_build_tree followed by tf_tree_mask: the same tree, mask,
position ids and status bits, bit for bit, with the mask written by the builder itself
(B + 1 <= 128) and by the separate mask kernel (larger trees)."""
import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu


def _both(cfg, corrupt_root=False):
    from paper_2606_03819_gb300 import Dims, Drafter
    from paper_2606_03819_gb300 import binding as B
    inp = synth.make_inputs(cfg)
    d = {k: v.cuda() for k, v in inp.items() if isinstance(v, torch.Tensor)}
    if corrupt_root:
        d["root_tok"][0] = cfg.V + 5
    dims = Dims.from_config(cfg)
    dr = Drafter(dims, d)
    dr.stage1(d["hidden"])
    if cfg.mode == "ar":
        dr.stage2(d["hidden"], d["root_tok"])
    n = cfg.B + 1
    sep = {k: torch.full((cfg.batch, n), 7, dtype=t, device="cuda") for k, t in
           (("tok", torch.int32), ("par", torch.int32), ("dep", torch.int32), ("score", torch.float32),
            ("pos", torch.int32))}
    sep["mask"] = torch.full((cfg.batch, n, n), 3, dtype=torch.uint8, device="cuda")
    sep["stat"] = torch.full((cfg.batch,), 9, dtype=torch.int32, device="cuda")
    fus = {k: torch.full_like(v, 5) for k, v in sep.items()}
    child_ids = dr.child_ids if cfg.mode == "ar" else None
    child_lp = dr.child_logp if cfg.mode == "ar" else None
    B.tf_build_tree(dims, d["root_tok"], dr.top_ids, dr.top_logp, child_ids, child_lp, sep["tok"], sep["par"],
                    sep["dep"], sep["score"], sep["stat"])
    B.tf_tree_mask(dims, sep["par"], sep["dep"], d["root_pos"], sep["mask"], sep["pos"])
    B.tf_build_tree_mask(dims, d["root_tok"], d["root_pos"], dr.top_ids, dr.top_logp, child_ids, child_lp,
                         fus["tok"], fus["par"], fus["dep"], fus["score"], fus["mask"], fus["pos"], fus["stat"])
    torch.cuda.synchronize()
    for k in sep:
        a, b = sep[k].cpu().numpy(), fus[k].cpu().numpy()
        if a.dtype == np.float32:
            np.testing.assert_array_equal(a.view(np.int32), b.view(np.int32), err_msg=k)
        else:
            np.testing.assert_array_equal(a, b, err_msg=k)
    return sep


@pytest.mark.parametrize("name,over", [
    ("tiny_peaked", dict(dtype="bf16", batch=3, V=2000)),                       # B + 1 = 13: fused
    ("tiny_peaked", dict(dtype="bf16", batch=2, V=2000, mode="marginal")),
    ("tiny_peaked", dict(dtype="bf16", batch=2, V=2000, mode="marginal_mary")),
    ("tiny_f32", dict(batch=2, B=127, K2=127)),                                 # B + 1 = 128: fused
    ("tiny_f32", dict(batch=2, B=128, K2=128)),                                 # B + 1 = 129: two launches
    ("tiny_f32", dict(batch=1, B=300, K2=64)),
])
def test_fused_mask_equals_separate_calls(name, over):
    _both(synth.get_config(name, **over))


def test_fused_mask_on_a_flagged_sequence():
    # an out-of-range root token is flagged, and the trees and masks still agree
    sep = _both(synth.get_config("tiny_peaked", dtype="bf16", batch=2, V=2000), corrupt_root=True)
    assert sep["stat"].cpu().numpy()[0] != 0
