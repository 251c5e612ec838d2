"""bench.py's roofline arithmetic on CPU: the LM-head pass is reported against HBM bandwidth
unless its contraction at the sustained tensor rate takes longer than streaming its bytes."""
import pytest

import bench
import synth

HBM = (6791.7, "measured")
TC = (1719.2, "measured")


def test_measured_shape_is_hbm_bound():
    cfg = synth.get_config("q8_b64")
    r = bench.lmhead_roofline(cfg, 16, cfg.R, 189.4e-3, 236.9e-3, HBM, TC, None, "t")
    assert r["bound"] == "hbm" and r["unit"] == "GB/s"
    # |W_lm| + the activation rows per launch, over the mean launch time
    b1 = cfg.V * cfg.d * 2 + 16 * cfg.d * 2
    b2 = cfg.V * cfg.d * 2 + 241 * cfg.d * 2
    assert r["bytes_per_launch"] == {"stage1": b1, "stage2": b2}
    assert r["achieved"] == pytest.approx((b1 + b2) / 2 / ((189.4e-3 + 236.9e-3) / 2 / 1e3) / 1e9)
    assert 0.85 < r["frac"] < 0.87


def test_two_token_shape_is_tensor_bound():
    cfg = synth.get_config("q8_b64_2prev")
    assert cfg.R == 3601
    r = bench.lmhead_roofline(cfg, 16, cfg.R, 193.3e-3, 2665.2e-3, HBM, TC, None, "t")
    assert r["bound"] == "tensor" and r["unit"] == "TFLOP/s"
    flops = 2.0 * (16 + 3601) * cfg.V * cfg.d
    assert r["achieved"] == pytest.approx(flops / 2 / ((193.3e-3 + 2665.2e-3) / 2 / 1e3) / 1e12)
    assert r["frac"] == pytest.approx(r["achieved"] / TC[0])
    assert r["hbm"]["unit"] == "GB/s" and r["hbm"]["frac"] < 0.2


def test_algorithmic_bytes_follow_the_approximator():
    base = bench.algorithmic_bytes(synth.get_config("q8_b64"))[0]
    lin = bench.algorithmic_bytes(synth.get_config("q8_b64_linear"))[0]
    two = bench.algorithmic_bytes(synth.get_config("q8_b64_2prev"))[0]
    d, I = 4096, 4096
    # SwiGLU 2 I 2d + d I weights; linear d 2d; two tokens 2 I 3d + d I and more gathered rows
    assert base - lin == (2 * I * 2 * d + d * I - d * 2 * d) * 2
    assert two - base == (2 * I * d) * 2 + (3601 - 241) * d * 2


def test_traffic_record_applies_to_its_own_workload_only():
    # the committed ncu record was scaled to the measured workload; other workloads get null
    rec = bench.profiled_traffic("q8_b64")
    assert rec is None or rec > 1.2e9
    assert bench.profiled_traffic("q8_b64_2prev") is None
    assert bench.profiled_traffic("q8_b6") is None


def test_torch_eager_reference_builds_the_oracles_tree():
    # the library-call reference point of bench.py computes the same tree as the oracle (fp32 on
    # the CPU here; on the GPU it runs in the workload's dtype)
    import numpy as np
    import torch

    import parity
    for batch, seed in ((1, 0), (3, 4)):
        cfg = synth.get_config("tiny_peaked", batch=batch, seed=seed)
        inp = synth.make_inputs(cfg)
        w = {k: v for k, v in inp.items() if isinstance(v, torch.Tensor)}
        trees = bench.torch_eager_tree(cfg, w, inp["hidden"], inp["root_tok"])
        orc = parity.run_oracle(cfg, inp)
        for s, (tok, par, dep, score) in enumerate(trees):
            np.testing.assert_array_equal(tok, orc[s].tree.tok)
            np.testing.assert_array_equal(par, orc[s].tree.parent)
            np.testing.assert_array_equal(dep, orc[s].tree.depth)
            np.testing.assert_allclose(score, orc[s].tree.score, atol=1e-4)
