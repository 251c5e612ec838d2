"""tf_stage1_marginals_static: the stage-1 LM-head top-k for callers that cannot allocate device
memory (a plugin inside a framework that owns all GPU memory and hands out no workspace, or a
latency-critical caller that must not call cudaMalloc/cudaFree because they can synchronise the
device). It uses a fixed scratch array inside the library instead of a caller's workspace.

Its results must equal those of tf_stage1_marginals (the workspace call) bit for bit on the same
inputs, because both run the same kernels on the same data, over two calls in a row with
different inputs: the shared array keeps the first call's contents, so a stale value would show
in the second. The size limit is checked on the host first.

This file is collected last on purpose (name order), after every other test."""
import ctypes
import os

import numpy as np
import pytest
import torch

def _lib():
    from paper_2606_03819_gb300 import binding
    if not os.path.exists(binding.LIB_PATH):
        from paper_2606_03819_gb300 import build
        build.build()
    return binding.load_library()


def _dims(**kw):
    from paper_2606_03819_gb300.binding import Dims
    base = dict(batch=1, d=128, V=2048, I=64, gamma=4, M=4, K2=12, B=12, dtype="f32", mode="marginal")
    base.update(kw)
    return Dims(**base)


def _call_static_raw(lib, dims, w_ptr=None, hidden=None, ids=None, logp=None, status=None):
    return lib.tf_stage1_marginals_static(ctypes.byref(dims.c()), w_ptr, hidden, ids, logp, status, None)


def test_static_entry_point_is_declared_and_exported():
    from paper_2606_03819_gb300 import binding
    lib = _lib()
    assert "tf_stage1_marginals_static" in binding.EXPORTS
    assert hasattr(lib, "tf_stage1_marginals_static")
    hdr = open(os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))),
                            "include", "treeflash.h")).read()
    assert "tf_stage1_marginals_static(" in hdr and "TF_STATIC_SCRATCH_BYTES" in hdr


def test_static_scratch_limit_is_checked_before_any_gpu_work():
    # Null pointers everywhere: a request beyond the scratch must fail on its size
    # (TF_ERR_UNSUPPORTED); one just inside must get as far as the pointer check
    # (TF_ERR_INVALID_ARG). Neither reaches the GPU.
    from paper_2606_03819_gb300 import binding as Bn
    lib = _lib()
    V = 151936                      # 594 blocks of 256, 160 bytes each per row: rows <= 88 fit in 8 MiB
    assert _call_static_raw(lib, _dims(batch=89, gamma=1, d=4096, V=V, dtype="bf16")) == Bn.TF_ERR_UNSUPPORTED
    assert _call_static_raw(lib, _dims(batch=30, gamma=3, d=4096, V=V, dtype="bf16")) == Bn.TF_ERR_UNSUPPORTED
    assert _call_static_raw(lib, _dims(batch=88, gamma=1, d=4096, V=V, dtype="bf16")) == Bn.TF_ERR_INVALID_ARG
    assert _call_static_raw(lib, _dims(batch=11, gamma=8, d=4096, V=V, dtype="bf16")) == Bn.TF_ERR_INVALID_ARG
    # invalid dims are rejected as by the workspace calls
    assert _call_static_raw(lib, _dims(V=8, K2=12)) == Bn.TF_ERR_INVALID_ARG
    assert _call_static_raw(lib, _dims(dtype="bf16", d=100)) == Bn.TF_ERR_UNSUPPORTED


def _weights(dims, gen, w_std=0.02):
    dt = dims.torch_dtype
    lm = (torch.randn(dims.V, dims.d, generator=gen, device="cuda") * w_std).to(dt)
    return {"lm_head": lm}


def _hidden(dims, gen, scale):
    dt = dims.torch_dtype
    return (torch.randn(dims.batch, dims.gamma, dims.d, generator=gen, device="cuda") * scale).to(dt)


def _workspace_result(dims, w, hidden):
    from paper_2606_03819_gb300 import binding as Bn
    ws = Bn.alloc_workspace(dims)
    ids = torch.empty(dims.batch, dims.gamma, dims.K1, dtype=torch.int32, device="cuda")
    lp = torch.empty(dims.batch, dims.gamma, dims.K1, dtype=torch.float32, device="cuda")
    Bn.tf_stage1_marginals(dims, w, hidden, ids, lp, ws)
    flags = Bn.tf_status_read(ws)
    return ids.cpu().numpy(), lp.cpu().numpy(), flags


def _static_result(dims, w, hidden):
    from paper_2606_03819_gb300 import binding as Bn
    ids = torch.full((dims.batch, dims.gamma, dims.K1), -7, dtype=torch.int32, device="cuda")
    lp = torch.full((dims.batch, dims.gamma, dims.K1), float("nan"), dtype=torch.float32, device="cuda")
    st = torch.full((1,), -1, dtype=torch.int32, device="cuda")
    Bn.tf_stage1_marginals_static(dims, w, hidden, ids, lp, st)
    torch.cuda.synchronize()
    return ids.cpu().numpy(), lp.cpu().numpy(), int(st.item())


def _compare(dims, ref, got, what):
    r_ids, r_lp, r_fl = ref
    g_ids, g_lp, g_fl = got
    assert np.isfinite(g_lp).all(), f"{what}: non-finite log-probabilities"
    np.testing.assert_array_equal(g_ids, r_ids, err_msg=f"{what}: token ids differ")
    # the same kernels on the same inputs: equal bit for bit
    np.testing.assert_array_equal(g_lp.view(np.uint32), r_lp.view(np.uint32),
                                  err_msg=f"{what}: log-probabilities differ")
    assert g_fl == r_fl, f"{what}: device flags {g_fl} != {r_fl}"
    assert not (g_fl & ~16), f"{what}: device flags {g_fl}"


CASES = [
    # fp32 CUDA-core path, ragged vocabulary, several row tiles
    ("f32", dict(batch=3, gamma=5, d=128, V=3001, M=4, K2=12, dtype="f32")),
    # bf16 tensor-core path, ragged vocabulary, 2 M-tiles of rows, k = 64
    ("bf16", dict(batch=4, gamma=40, d=256, V=5003, M=8, K2=64, dtype="bf16")),
]


@pytest.mark.gpu
@pytest.mark.parametrize("name,kw", CASES, ids=[c[0] for c in CASES])
def test_static_matches_workspace_call_on_two_calls_in_a_row(name, kw):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    _lib()
    dims = _dims(**kw)
    gen = torch.Generator(device="cuda").manual_seed(1234)
    w = _weights(dims, gen)
    # two different inputs: peaked, then flat marginals
    scale_peaked = 6.0 / (0.02 * dims.d ** 0.5)
    scale_flat = 1.0 / (0.02 * dims.d ** 0.5)
    for call, scale in enumerate((scale_peaked, scale_flat)):
        hidden = _hidden(dims, gen, scale)
        ref = _workspace_result(dims, w, hidden)
        got = _static_result(dims, w, hidden)
        _compare(dims, ref, got, f"{name} call {call + 1}")


@pytest.mark.gpu
def test_static_at_its_size_limit():
    # the largest request the scratch holds at the 151936-entry vocabulary: 88 rows
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    _lib()
    dims = _dims(batch=11, gamma=8, d=4096, V=151936, M=8, K2=32, dtype="bf16")
    gen = torch.Generator(device="cuda").manual_seed(99)
    w = _weights(dims, gen)
    for call in range(2):
        hidden = _hidden(dims, gen, (2.0 + call) / (0.02 * dims.d ** 0.5))
        _compare(dims, _workspace_result(dims, w, hidden), _static_result(dims, w, hidden),
                 f"limit call {call + 1}")
    del w
    torch.cuda.empty_cache()
