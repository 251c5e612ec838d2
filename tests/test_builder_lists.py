"""Part 2 of Algorithm 1 on hand-made child lists: tf_build_tree against the oracle's lazy queue,
bit for bit (tokens, parents, depths, scores, status). Log-probabilities are multiples of 1/8 in
[-6, 0], so every path score is exact in fp32 and fp64 alike and equal scores are frequent (the
tie rules decide many pops); a random share of every list's tokens are stage-1 candidates of the
list's depth, so the M-ary rule expands often and the trees grow deep and wide. Budgets up to 64
run the sorted-queue builder, larger ones the register and shared-memory builders."""
import numpy as np
import pytest
import torch

import oracle.treeflash_oracle as O

pytestmark = pytest.mark.gpu

BACKGROUND = -1.0e6   # every token outside a list: below every listed value


def _sorted_list(rng, ids, V):
    vals = -rng.integers(0, 49, ids.shape[0]).astype(np.float64) / 8.0 + 0.0   # no -0.0
    order = np.lexsort((ids, -vals))        # larger value first, equal values by smaller id
    return ids[order], vals[order]


def _list_tokens(rng, n, V, cands):
    """n distinct tokens of [0, V), a random number of them from `cands`."""
    cands = np.unique(cands)
    n_c = int(rng.integers(0, min(n, cands.shape[0]) + 1))
    chosen = rng.choice(cands, n_c, replace=False) if n_c else np.zeros(0, np.int64)
    rest = np.setdiff1d(np.arange(V), chosen)
    return np.concatenate([chosen, rng.choice(rest, n - n_c, replace=False)]).astype(np.int64)


def _make(rng, mode, b, gamma, M, K2, V):
    K1 = max(M, K2)
    R = 1 + M * (gamma - 1)
    top_ids = np.zeros((b, gamma, K1), np.int64)
    top_lp = np.zeros((b, gamma, K1))
    child_ids = np.zeros((b, R, K2), np.int64)
    child_lp = np.zeros((b, R, K2))
    for s in range(b):
        for i in range(gamma):
            prev = top_ids[s, i - 1, :M] if i > 0 else np.zeros(0, np.int64)
            top_ids[s, i], top_lp[s, i] = _sorted_list(rng, _list_tokens(rng, K1, V, prev), V)
        for r in range(R):
            dep = 1 if r == 0 else (r - 1) // M + 2          # depth of the row's entries (reading R4)
            ids = _list_tokens(rng, K2, V, top_ids[s, dep - 1, :M])
            child_ids[s, r], child_lp[s, r] = _sorted_list(rng, ids, V)
    root = rng.integers(0, V, b)
    return top_ids, top_lp, child_ids, child_lp, root


def _full_rows(ids, lp, V):
    rows = np.full((ids.shape[0], V), BACKGROUND)
    for r in range(ids.shape[0]):
        rows[r, ids[r]] = lp[r]
    return rows


CASES = [
    # mode, batch, gamma, M, K2, B, V
    ("ar", 4, 16, 16, 64, 64, 5000),       # the Qwen3-8B-shaped B = 64 tree
    ("ar", 4, 16, 8, 32, 32, 3000),
    ("ar", 3, 16, 16, 64, 63, 2000),
    ("ar", 3, 6, 3, 12, 20, 500),          # M not a multiple of 4, K2 < B truncates the lists
    ("ar", 3, 5, 6, 40, 64, 300),
    ("ar", 2, 4, 1, 8, 10, 100),
    ("ar", 2, 16, 64, 64, 64, 4000),       # M = 64
    ("ar", 2, 3, 2, 4, 30, 50),            # underfull universe
    ("marginal", 3, 8, 4, 64, 64, 1000),
    ("marginal_mary", 3, 8, 5, 16, 40, 1000),
    ("ar", 2, 8, 8, 100, 100, 3000),       # register builder
    ("ar", 1, 8, 8, 64, 200, 3000),        # shared-memory builder, K2 < B
]


@pytest.mark.parametrize("mode,b,gamma,M,K2,B,V", CASES)
def test_builder_equals_the_oracle_on_hand_made_lists(mode, b, gamma, M, K2, B, V):
    from paper_2606_03819_gb300 import Dims
    from paper_2606_03819_gb300 import binding as Bn
    dims = Dims(b, 64, V, 64, gamma, M, K2, B, dtype="f32", mode=mode)
    n = B + 1
    for seed in range(6):
        rng = np.random.default_rng(1000 * seed + 7 * B + M)
        top_ids, top_lp, child_ids, child_lp, root = _make(rng, mode, b, gamma, M, K2, V)
        dev = lambda a, t: torch.from_numpy(np.ascontiguousarray(a)).to(device="cuda", dtype=t)
        out = {k: torch.full((b, n), -7, dtype=t, device="cuda") for k, t in
               (("tok", torch.int32), ("par", torch.int32), ("dep", torch.int32), ("score", torch.float32))}
        stat = torch.full((b,), -7, dtype=torch.int32, device="cuda")
        ar = mode == "ar"
        Bn.tf_build_tree(dims, dev(root, torch.int32), dev(top_ids, torch.int32), dev(top_lp, torch.float32),
                         dev(child_ids, torch.int32) if ar else None, dev(child_lp, torch.float32) if ar else None,
                         out["tok"], out["par"], out["dep"], out["score"], stat)
        torch.cuda.synchronize()
        got = {k: v.cpu().numpy() for k, v in out.items()}
        st = stat.cpu().numpy()
        for s in range(b):
            s1 = _full_rows(top_ids[s], top_lp[s], V)
            s2 = _full_rows(child_ids[s], child_lp[s], V) if ar else None
            src = O.ChildSource(mode, gamma, M, top_ids[s], s1, s2)
            t = O.build_tree_lazy(src, int(root[s]), B, keep=K2 if K2 < B else None)
            where = f"seed {seed} sequence {s}"
            np.testing.assert_array_equal(got["tok"][s], t.tok, err_msg=where)
            np.testing.assert_array_equal(got["par"][s], t.parent, err_msg=where)
            np.testing.assert_array_equal(got["dep"][s], t.depth, err_msg=where)
            np.testing.assert_array_equal(got["score"][s].astype(np.float64), t.score, err_msg=where)
            assert st[s] == (O_UNDERFULL if t.underfull else 0), where


O_UNDERFULL = 2   # TF_DEV_UNDERFULL
