"""tf_draft_tree_host on a created stream with page-locked buffers: the first call captures the step
as a CUDA graph, later calls with the same arguments replay it. Each call must give the device
path's tree, mask, position ids and status on the inputs the host buffers hold at that call, the
same return code, and add the same number of kernel launches to the library's counter."""
import numpy as np
import pytest
import torch

import parity
import synth

pytestmark = pytest.mark.gpu

OUT = (("node_tok", torch.int32), ("node_parent", torch.int32), ("node_depth", torch.int32),
       ("node_score", torch.float32), ("pos_ids", torch.int32))


def _host_buffers(cfg):
    n = cfg.B + 1
    out = {k: torch.empty(cfg.batch, n, dtype=t).pin_memory() for k, t in OUT}
    out["mask"] = torch.empty(cfg.batch, n, n, dtype=torch.uint8).pin_memory()
    out["dev_status"] = torch.empty(cfg.batch, dtype=torch.int32).pin_memory()
    return out


def _call(Bn, dims, d, h, out, ws, stream):
    return Bn.tf_draft_tree_host(dims, d, h["hidden"], h["root_tok"], h["root_pos"], out["node_tok"],
                                 out["node_parent"], out["node_depth"], out["node_score"], out["mask"],
                                 out["pos_ids"], out["dev_status"], ws, stream=stream)


@pytest.mark.parametrize("name,over", [
    ("tiny_peaked", dict(dtype="bf16", batch=3, V=2000)),
    ("tiny_peaked", dict(dtype="bf16", batch=2, V=2000, mode="marginal")),
    ("tiny_f32", dict(batch=2, B=200, K2=64)),                  # B + 1 > 128: the separate mask kernel
])
def test_replayed_step_equals_the_device_path(name, over):
    from paper_2606_03819_gb300 import Dims, alloc_workspace
    from paper_2606_03819_gb300 import binding as Bn
    cfg = synth.get_config(name, **over)
    dims = Dims.from_config(cfg)
    base = synth.make_inputs(cfg)
    d = parity.device_inputs(base)
    h = {k: base[k].clone().pin_memory() for k in ("hidden", "root_tok", "root_pos")}
    out = _host_buffers(cfg)
    ws = alloc_workspace(dims)
    stream = torch.cuda.Stream()
    launches = []
    for call in range(3):
        # new contents in the same page-locked buffers: the replayed graph reads them
        g = torch.Generator().manual_seed(100 + call)
        h["hidden"].copy_(base["hidden"] * (1.0 + 0.25 * torch.rand((), generator=g)))
        h["root_tok"].copy_(torch.randint(0, cfg.V, h["root_tok"].shape, generator=g, dtype=h["root_tok"].dtype))
        if call == 2:
            h["root_tok"][0] = cfg.V + 3                       # a bad root token: flagged, not fatal
        n0 = Bn.tf_kernel_launches()
        st = _call(Bn, dims, d, h, out, ws, stream)
        launches.append(Bn.tf_kernel_launches() - n0)
        dev_in = dict(d, hidden=h["hidden"].cuda(), root_tok=h["root_tok"].cuda(), root_pos=h["root_pos"].cuda())
        ref = parity.run_gpu(cfg, dev_in)
        for k in ("node_tok", "node_parent", "node_depth", "mask", "pos_ids"):
            np.testing.assert_array_equal(out[k].numpy(), ref[k], err_msg=f"call {call}: {k}")
        np.testing.assert_array_equal(out["node_score"].numpy().view(np.int32), ref["node_score"].view(np.int32))
        # dev_status: the sequence's bits OR-ed with the workspace status word, nothing else
        np.testing.assert_array_equal(out["dev_status"].numpy(), ref["dev_status"] | ref["flags"])
        expect = Bn.TF_ERR_DEVICE_STATUS if ref["flags"] & ~16 else Bn.TF_OK
        assert st == expect, (call, st, ref["flags"])
    assert launches[1] == launches[2] == launches[0] > 0
