"""The verification walk (tf_accept_walk) against the oracle's walk: acceptance by an equality
check with the verifier's tokens (Sec. 3) and the step's block efficiency (Sec. 4), on trees the
GPU path builds and on hand-made trees with missing nodes, for verifier tokens that agree with
the tree along random, full-depth and empty paths. Results are integer: compared bit for bit."""
import ctypes

import numpy as np
import pytest
import torch

import synth
from oracle import treeflash_oracle as O

import parity  # noqa: E402  (tests/ is on sys.path)


def _lib():
    import os
    from paper_2606_03819_gb300 import binding
    if not os.path.exists(binding.LIB_PATH):
        from paper_2606_03819_gb300 import build
        build.build()
    return binding.load_library()


def test_accept_walk_rejects_missing_arguments_before_gpu_work():
    from paper_2606_03819_gb300 import binding as Bn
    lib = _lib()
    dims = Bn.Dims(batch=1, d=128, V=2048, I=64, gamma=4, M=4, K2=12, B=12, dtype="f32", mode="ar")
    st = lib.tf_accept_walk(ctypes.byref(dims.c()), None, None, None, None, None, None, None)
    assert st == Bn.TF_ERR_INVALID_ARG


def _verifier_tokens(tok, par, rng, mode):
    """Verifier tokens per node: 'random' agrees with a random child with probability 0.7,
    'deep' agrees along the deepest path, 'none' never agrees."""
    n = len(tok)
    children = {i: [c for c in range(1, n) if par[c] == i] for i in range(n)}
    ver = np.full(n, 0, dtype=np.int64)
    for i in range(n):
        ver[i] = 900_000 + i                                  # a token no node carries
    if mode == "random":
        for i in range(n):
            if children[i] and rng.random() < 0.7:
                ver[i] = tok[rng.choice(children[i])]
    elif mode == "deep":
        depth = np.zeros(n, dtype=np.int64)
        for i in range(1, n):
            if par[i] >= 0:
                depth[i] = depth[par[i]] + 1
        j = int(np.argmax(np.where(par >= 0, depth, -1) if n > 1 else depth))
        while j > 0:
            ver[par[j]] = tok[j]
            j = int(par[j])
    return ver


def _run_walk(dims, tok, par, ver):
    from paper_2606_03819_gb300 import binding as Bn
    b, n = tok.shape
    t = torch.from_numpy(tok.astype(np.int32)).cuda()
    p = torch.from_numpy(par.astype(np.int32)).cuda()
    v = torch.from_numpy(ver.astype(np.int32)).cuda()
    alen = torch.full((b,), -7, dtype=torch.int32, device="cuda")
    apath = torch.full((b, dims.gamma + 1), -7, dtype=torch.int32, device="cuda")
    nxt = torch.full((b,), -7, dtype=torch.int32, device="cuda")
    Bn.tf_accept_walk(dims, t, p, v, alen, apath, nxt)
    torch.cuda.synchronize()
    return alen.cpu().numpy(), apath.cpu().numpy(), nxt.cpu().numpy()


def _check(dims, tok, par, ver):
    alen, apath, nxt = _run_walk(dims, tok, par, ver)
    taus = []
    for s in range(tok.shape[0]):
        path, bonus = O.accept_walk(tok[s], par[s], ver[s])
        assert alen[s] == len(path) - 1, f"seq {s}: accepted {alen[s]} vs {len(path) - 1}"
        assert apath[s, :len(path)].tolist() == path, f"seq {s}: path"
        assert (apath[s, len(path):] == -1).all()
        assert nxt[s] == bonus, f"seq {s}: bonus token"
        taus.append(len(path))
    return taus


@pytest.mark.gpu
@pytest.mark.parametrize("mode", ["random", "deep", "none"])
def test_accept_walk_matches_the_oracle_on_gpu_trees(mode):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    _lib()
    from paper_2606_03819_gb300 import binding as Bn
    cfg = synth.get_config("tiny_peaked", dtype="bf16", batch=6, V=2000, B=24, K2=24, gamma=6, M=4)
    gpu = parity.run_gpu(cfg, parity.device_inputs(synth.make_inputs(cfg)))
    tok, par = gpu["node_tok"].astype(np.int64), gpu["node_parent"].astype(np.int64)
    rng = np.random.default_rng({"random": 1, "deep": 2, "none": 3}[mode])
    ver = np.stack([_verifier_tokens(tok[s], par[s], rng, mode) for s in range(cfg.batch)])
    taus = _check(Bn.Dims.from_config(cfg), tok, par, ver)
    if mode == "none":
        assert taus == [1] * cfg.batch
    if mode == "deep":
        assert all(t >= 2 for t in taus)


@pytest.mark.gpu
def test_accept_walk_on_trees_with_missing_nodes_and_full_depth():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    _lib()
    from paper_2606_03819_gb300 import binding as Bn
    dims = Bn.Dims(batch=3, d=128, V=64, I=64, gamma=4, M=4, K2=8, B=8, dtype="f32", mode="ar")
    # seq 0: a chain of depth 4 (the depth cap) fully accepted; seq 1: missing nodes (an
    # underfull tree) whose tokens would match; seq 2: the verifier agrees with node 2, not 1
    tok = np.array([[50, 1, 2, 3, 4, 5, -1, -1, -1],
                    [50, 7, 8, 33, 33, -1, -1, -1, -1],
                    [50, 7, 8, 9, 10, 11, 12, 13, 14]])
    par = np.array([[-1, 0, 1, 2, 3, 0, -1, -1, -1],
                    [-1, 0, 0, -1, -1, -1, -1, -1, -1],
                    [-1, 0, 0, 1, 2, 2, 4, 5, 6]])
    ver = np.array([[1, 2, 3, 4, 99, 0, 0, 0, 0],
                    [7, 33, 0, 0, 0, 0, 0, 0, 0],
                    [8, 9, 11, 0, 0, 0, 0, 0, 0]])
    taus = _check(dims, tok, par, ver)
    assert taus == [5, 2, 3]
