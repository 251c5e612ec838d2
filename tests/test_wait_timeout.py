"""Failure detection without a GPU fault: every wait of the tensor-core kernels is bounded.

With the progress-wait limit set far below a copy's latency (tf_set_wait_limit_ns), the
LM-head kernel must give up, set TF_DEV_TIMEOUT (tf_status_read -> TF_ERR_TIMEOUT), drain its
own copies and MMAs and return, leaving the context usable: a following call with the default
limit on the same stream must give the results of a call made before, bit for bit. Covered for
one CTA per tile (16 rows) and for CTA pairs (200 rows, two M-tiles). The timed-out call's
partials are never merged."""
import pytest
import torch

from paper_2606_03819_gb300 import binding as Bn


def test_wait_limit_setter_checks_its_range():
    Bn.load_library()
    with pytest.raises(Bn.TreeFlashError):
        Bn.tf_set_wait_limit_ns(61 * 10 ** 9)
    Bn.tf_set_wait_limit_ns(0)


def _lmhead(dims, lm, x, rows, ws):
    ids = torch.empty(rows, dims.K1, dtype=torch.int32, device="cuda")
    lp = torch.empty(rows, dims.K1, dtype=torch.float32, device="cuda")
    Bn.tf_status_reset(ws)
    Bn.tf_lmhead_partials(dims, lm, x, rows, ws)
    Bn.tf_lmhead_merge(dims, lm, x, rows, dims.K1, ids, lp, ws)
    return ids.cpu(), lp.cpu(), Bn.tf_status_read(ws)


@pytest.mark.gpu
@pytest.mark.parametrize("batch,gamma", [(1, 16), (4, 50)], ids=["one_cta_per_tile", "cta_pairs"])
def test_bounded_wait_times_out_and_the_context_stays_usable(batch, gamma):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    Bn.load_library()
    dims = Bn.Dims(batch=batch, d=4096, V=4096, I=64, gamma=gamma, M=4, K2=8, B=8, dtype="bf16",
                   mode="marginal")
    rows = batch * gamma
    gen = torch.Generator(device="cuda").manual_seed(7)
    lm = (torch.randn(dims.V, dims.d, generator=gen, device="cuda") * 0.02).to(torch.bfloat16)
    x = (torch.randn(rows, dims.d, generator=gen, device="cuda") * 2.0).to(torch.bfloat16)
    ws = Bn.alloc_workspace(dims)
    try:
        Bn.tf_set_wait_limit_ns(0)
        ref_ids, ref_lp, flags = _lmhead(dims, lm, x, rows, ws)
        assert not (flags & ~Bn.TF_DEV_RECOMPUTED), f"reference call flags {flags}"
        # 1 ns: any wait that is not satisfied within its first polls gives up (64 K-steps per
        # vocabulary block stream through a ring of a few stages, so many waits are real)
        Bn.tf_set_wait_limit_ns(1)
        Bn.tf_status_reset(ws)
        Bn.tf_lmhead_partials(dims, lm, x, rows, ws)
        flags = Bn.tf_status_read(ws)
        assert flags & Bn.TF_DEV_TIMEOUT, f"no timeout reported (flags {flags})"
        torch.cuda.synchronize()     # no sticky error: the kernel returned normally
        # back to the default limit, same stream and workspace: the call must be exact again
        Bn.tf_set_wait_limit_ns(0)
        ids, lp, flags = _lmhead(dims, lm, x, rows, ws)
        assert not (flags & ~Bn.TF_DEV_RECOMPUTED), f"call after the timeout: flags {flags}"
        assert torch.equal(ids, ref_ids)
        assert torch.equal(lp.view(torch.int32), ref_lp.view(torch.int32))
    finally:
        Bn.tf_set_wait_limit_ns(0)
