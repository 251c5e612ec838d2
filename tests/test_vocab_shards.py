"""The vocabulary-parallel split of the LM head (one exchange step after each LM-head pass),
simulated on one GPU: each shard of W_lm (a multiple of 256 rows) runs the LM-head pass alone;
exchanging the partial tables (the block ranges side by side, half-block best ids shifted by
the shard's first token) and merging once must give exactly the unsharded top-k and log-probs.
A P-rank run would all-gather these tables; every run here has one GPU."""
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import os
    from paper_2606_03819_gb300 import binding
    if not os.path.exists(binding.LIB_PATH):
        from paper_2606_03819_gb300 import build
        build.build()
    binding.load_library()


def _dims(V, dtype, rows_b, gamma, K2):
    from paper_2606_03819_gb300.binding import Dims
    return Dims(batch=rows_b, d=256, V=V, I=64, gamma=gamma, M=4, K2=K2, B=K2, dtype=dtype, mode="marginal")


@pytest.mark.parametrize("dtype,shards", [("bf16", (1024, 2048, 1280)), ("f32", (2048, 2048))])
def test_sharded_partials_merge_to_the_unsharded_topk(dtype, shards):
    from paper_2606_03819_gb300 import binding as Bn
    V = sum(shards)
    b, gamma, k = 3, 5, 48
    rows = b * gamma
    full = _dims(V, dtype, b, gamma, k)
    g = torch.Generator().manual_seed(7)
    dt = full.torch_dtype
    W = (torch.randn(V, full.d, generator=g) * 0.02).to(dt).cuda()
    x = (torch.randn(rows, full.d, generator=g) * 30.0).to(dt).cuda()
    ids0 = torch.empty(rows, k, dtype=torch.int32, device="cuda")
    lp0 = torch.empty(rows, k, dtype=torch.float32, device="cuda")
    ws = Bn.alloc_workspace(full)
    Bn.tf_status_reset(ws)
    Bn.tf_lmhead_partials(full, W, x, rows, ws)
    Bn.tf_lmhead_merge(full, W, x, rows, k, ids0, lp0, ws)
    assert not (Bn.tf_status_read(ws) & ~16)
    ref_h = Bn.tf_workspace_view(full, ws, Bn.TF_VIEW_HALVES, rows).clone()
    ref_c = Bn.tf_workspace_view(full, ws, Bn.TF_VIEW_CHUNKS, rows).clone()

    # each shard alone, then the exchange into one table
    halves, chunks = [], []
    v0 = 0
    for Vp in shards:
        dp = _dims(Vp, dtype, b, gamma, k)
        wsp = Bn.alloc_workspace(dp)
        Bn.tf_lmhead_partials(dp, W[v0:v0 + Vp], x, rows, wsp)
        h = Bn.tf_workspace_view(dp, wsp, Bn.TF_VIEW_HALVES, rows).clone()
        c = Bn.tf_workspace_view(dp, wsp, Bn.TF_VIEW_CHUNKS, rows).clone()
        hid = h[..., 3].view(torch.int32)
        hid[hid >= 0] += v0                     # half-block best ids become global token ids
        halves.append(h)
        chunks.append(c)
        v0 += Vp
    H, C = torch.cat(halves, 0), torch.cat(chunks, 0)
    assert torch.equal(H, ref_h) and torch.equal(C, ref_c), "per-shard partials differ from the unsharded pass"

    # merge the exchanged table
    Bn.tf_workspace_view(full, ws, Bn.TF_VIEW_HALVES, rows).copy_(H)
    Bn.tf_workspace_view(full, ws, Bn.TF_VIEW_CHUNKS, rows).copy_(C)
    ids1 = torch.empty_like(ids0)
    lp1 = torch.empty_like(lp0)
    Bn.tf_lmhead_merge(full, W, x, rows, k, ids1, lp1, ws)
    torch.cuda.synchronize()
    assert torch.equal(ids1, ids0) and torch.equal(lp1, lp0)
    assert (ids0 >= 0).all()
