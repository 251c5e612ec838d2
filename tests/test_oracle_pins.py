"""Pins of the fp64 oracle against facts the paper and the mathematics fix (no GPU).

Each test names what pins it: a closed form, a library routine computing the same
definition independently, an invariant stated in the paper, or brute-force enumeration.
A plausible slip in the oracle (a dropped term, a wrong index or sign, a transposed
operand, a wrong tie rule) makes at least one of these fail.
"""
import itertools
import math

import numpy as np
import pytest
import scipy.special
import torch

from oracle import treeflash_oracle as O


def small_problem(V=32, d=16, I=24, gamma=4, seed=0, h_scale=3.0, wd_std=0.3, w_std=0.3):
    rng = np.random.default_rng(seed)
    W = dict(lm_head=rng.normal(0, w_std, (V, d)), embed=rng.normal(0, 1.0, (V, d)),
             norm_h=rng.uniform(0.5, 1.5, d), norm_e=rng.uniform(0.5, 1.5, d),
             w_gate=rng.normal(0, w_std, (I, 2 * d)), w_up=rng.normal(0, w_std, (I, 2 * d)),
             w_down=rng.normal(0, wd_std, (d, I)))
    H = rng.normal(0, h_scale, (gamma, d))
    root = int(rng.integers(0, V))
    return H, root, W


# ------------------------------------------------------------------ elementary pieces


def test_bf16_round_matches_torch_on_float32_values():
    # pinned to torch's float32 -> bfloat16 conversion (round to nearest even)
    x = np.random.default_rng(1).normal(0, 10, 20000).astype(np.float32)
    x = np.concatenate([x, np.float32([1.0, -2.5, 3.0e-3, 65504.0])])
    ours = O.bf16_round(x.astype(np.float64))
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(ours, ref)


def test_bf16_round_ties_to_even():
    # 1 + 2^-8 lies halfway between 1 and 1 + 2^-7: the even neighbour is 1.
    # 1 + 3*2^-8 lies halfway between 1 + 2^-7 and 1 + 2^-6: the even neighbour is 1 + 2^-6.
    assert O.bf16_round(np.array([1 + 2.0 ** -8]))[0] == 1.0
    assert O.bf16_round(np.array([1 + 3 * 2.0 ** -8]))[0] == 1 + 2.0 ** -6
    assert O.bf16_round(np.array([-(1 + 2.0 ** -8)]))[0] == -1.0


def test_rmsnorm_closed_form():
    # constant vector c*1: mean(x^2) = c^2, so every entry is c / sqrt(c^2 + eps) * w
    c, eps = 0.7, 1e-3
    w = np.array([1.0, 2.0, -1.0, 0.5])
    y = O.rmsnorm(np.full(4, c), w, eps)
    np.testing.assert_allclose(y, c / math.sqrt(c * c + eps) * w, rtol=1e-15)
    # scale invariance when eps = 0
    x = np.random.default_rng(2).normal(size=9)
    np.testing.assert_allclose(O.rmsnorm(5 * x, np.ones(9), 0.0), O.rmsnorm(x, np.ones(9), 0.0))
    # the result has unit root-mean-square when w = 1 and eps = 0
    assert abs(np.sqrt(np.mean(O.rmsnorm(x, np.ones(9), 0.0) ** 2)) - 1) < 1e-14


def test_silu_against_scipy_expit():
    x = np.linspace(-30, 30, 601)
    np.testing.assert_allclose(O.silu(x), x * scipy.special.expit(x), rtol=1e-13, atol=1e-300)
    assert O.silu(np.array([0.0]))[0] == 0.0


def test_log_softmax_sums_to_one_and_matches_scipy():
    z = np.random.default_rng(3).normal(0, 8, (5, 1000))
    lp = O.log_softmax(z)
    np.testing.assert_allclose(np.exp(lp).sum(axis=1), 1.0, rtol=1e-13)
    np.testing.assert_allclose(lp, scipy.special.log_softmax(z, axis=1), atol=1e-12)
    # shift invariance
    np.testing.assert_allclose(O.log_softmax(z + 123.0), lp, atol=1e-10)


def test_ranked_tie_rule():
    v = np.array([1.0, 3.0, 3.0, 2.0, 3.0, 1.0])
    # larger value first, then smaller index (reading R8)
    assert list(O.ranked(v)) == [1, 2, 4, 3, 0, 5]
    assert list(O.ranked(v, 2)) == [1, 2]
    # against an explicit sort by the composite key
    x = np.random.default_rng(4).integers(0, 5, 200).astype(float)
    assert list(O.ranked(x)) == sorted(range(200), key=lambda i: (-x[i], i))


def test_lm_head_orientation_and_temperature():
    # z_v = <W_lm[v], x> / T: one-hot x picks column k of W_lm
    W = np.arange(12.0).reshape(4, 3)
    x = np.array([[0.0, 1.0, 0.0]])
    np.testing.assert_array_equal(O.lm_head(x, W, 1.0)[0], W[:, 1])
    np.testing.assert_array_equal(O.lm_head(x, W, 2.0)[0], W[:, 1] / 2)


# ------------------------------------------------------------------ stage 1


def test_stage1_topk_matches_torch_topk():
    H, _, W = small_problem(V=500, d=24, gamma=3, seed=5)
    logp, ids, lp = O.stage1(H, W["lm_head"], 1.0, 7)
    z = torch.from_numpy(H) @ torch.from_numpy(W["lm_head"]).T
    tv, ti = torch.topk(z, 7, dim=1)
    np.testing.assert_array_equal(ids, ti.numpy())
    np.testing.assert_allclose(lp, torch.log_softmax(z, dim=1).gather(1, ti).numpy(), atol=1e-12)
    np.testing.assert_allclose(np.exp(logp).sum(1), 1.0, rtol=1e-13)


# ------------------------------------------------------------------ Eq. 1 and stage 2


def test_stage2_row_layout():
    gamma, M = 5, 3
    top = np.arange(gamma * 10).reshape(gamma, 10)
    hid, prev = O.stage2_conditioning(gamma, M, root_tok=77, top_ids=top)
    assert len(hid) == 1 + M * (gamma - 1)             # reading R4
    assert hid[0] == 0 and prev[0] == 77               # depth 1 conditioned on the root
    for i in range(2, gamma + 1):
        for m in range(M):
            r = 1 + (i - 2) * M + m
            assert hid[r] == i - 1                     # refines h_{t+i}
            assert prev[r] == top[i - 2, m]            # on candidate m of depth i-1


def test_ar_approximator_hand_computed():
    # d = 2, I = 1. norm weights 1, eps = 0.
    # h = (3, 4): RMS = sqrt(12.5); e = (1, -1): RMS = 1.
    # x = (3, 4)/sqrt(12.5) :: (1, -1)
    h = np.array([[3.0, 4.0]])
    e = np.array([[1.0, -1.0]])
    wg = np.array([[1.0, 0.0, 1.0, 0.0]])   # G = x0 + x2
    wu = np.array([[0.0, 1.0, 0.0, -1.0]])  # U = x1 - x3
    wd = np.array([[2.0], [-1.0]])
    x0, x1 = 3 / math.sqrt(12.5), 4 / math.sqrt(12.5)
    G, U = x0 + 1.0, x1 + 1.0
    a = G / (1 + math.exp(-G)) * U
    expect = np.array([[3 + 2 * a, 4 - a]])
    got = O.ar_approximator(h, e, np.ones(2), np.ones(2), wg, wu, wd, 0.0)
    np.testing.assert_allclose(got, expect, rtol=1e-14)


def test_zero_w_down_gives_identity():
    # zero-initialised approximator (training start, Sec. 3 "Training"): h' = h
    H, root, W = small_problem(seed=6)
    W["w_down"][:] = 0.0
    _, ids, _ = O.stage1(H, W["lm_head"], 1.0, 4)
    hp, lp = O.stage2(H, root, ids, W, 3, 1.0, 1e-6)
    hid, _ = O.stage2_conditioning(H.shape[0], 3, root, ids)
    np.testing.assert_array_equal(hp, H[hid])
    np.testing.assert_allclose(np.exp(lp).sum(1), 1.0, rtol=1e-13)


def test_concat_order_hidden_first():
    # x = [h~ ; e] (Eq. 1, h~ first). Zeroing the second half of W_gate and W_up removes the
    # token dependence, so the M rows of a depth coincide; zeroing the first half instead
    # makes rows that share a previous token but refine different depths differ only in h.
    H, root, W = small_problem(seed=7, gamma=3)
    d = H.shape[1]
    _, ids, _ = O.stage1(H, W["lm_head"], 1.0, 4)
    Wh = dict(W, w_gate=W["w_gate"].copy(), w_up=W["w_up"].copy())
    Wh["w_gate"][:, d:] = 0.0
    Wh["w_up"][:, d:] = 0.0
    hp, _ = O.stage2(H, root, ids, Wh, 3, 1.0, 1e-6)
    np.testing.assert_allclose(hp[1:4], np.repeat(hp[1:2], 3, axis=0), atol=1e-12)
    hp_full, _ = O.stage2(H, root, ids, W, 3, 1.0, 1e-6)
    assert np.abs(hp_full[1] - hp_full[2]).max() > 1e-3
    We = dict(W, w_gate=W["w_gate"].copy(), w_up=W["w_up"].copy())
    We["w_gate"][:, :d] = 0.0
    We["w_up"][:, :d] = 0.0
    hpe, _ = O.stage2(H, root, ids, We, 3, 1.0, 1e-6)
    hid, prev = O.stage2_conditioning(3, 3, root, ids)
    # delta = h' - h depends on the previous token only
    delta = hpe - H[hid]
    for a in range(len(prev)):
        for b in range(len(prev)):
            if prev[a] == prev[b]:
                np.testing.assert_allclose(delta[a], delta[b], atol=1e-12)


def test_linear_approximator_hand_computed():
    # "w/ Linear" ablation (Sec. 4, Table 3; reading R12): h' = h + W_lin [h~ ; e].
    # d = 2, norm weights 1, eps = 0; h = (3, 4): RMS sqrt(12.5); e = (1, -1): RMS 1.
    h = np.array([[3.0, 4.0]])
    e = np.array([[1.0, -1.0]])
    w_lin = np.array([[1.0, 0.0, 2.0, 0.0],     # out0 = x0 + 2 x2
                      [0.0, -1.0, 0.0, 3.0]])   # out1 = -x1 + 3 x3
    x0, x1 = 3 / math.sqrt(12.5), 4 / math.sqrt(12.5)
    expect = np.array([[3 + x0 + 2.0, 4 - x1 - 3.0]])
    got = O.linear_approximator(h, e, np.ones(2), np.ones(2), w_lin, 0.0)
    np.testing.assert_allclose(got, expect, rtol=1e-14)


def test_linear_approximator_identity_blocks():
    # W_lin = [I | 0] adds the normalised hidden state, [0 | I] the normalised embedding:
    # pins which half of the input is which (h~ first) against rmsnorm's closed form.
    rng = np.random.default_rng(9)
    d = 6
    h, e = rng.normal(0, 2, (3, d)), rng.normal(0, 1, (3, d))
    wh, we = rng.uniform(0.5, 1.5, d), rng.uniform(0.5, 1.5, d)
    eye, zero = np.eye(d), np.zeros((d, d))
    eps = 1e-6
    rms = lambda a: np.sqrt((a * a).mean(axis=1, keepdims=True) + eps)
    got_h = O.linear_approximator(h, e, wh, we, np.hstack([eye, zero]), eps)
    got_e = O.linear_approximator(h, e, wh, we, np.hstack([zero, eye]), eps)
    np.testing.assert_allclose(got_h, h + h / rms(h) * wh, rtol=1e-13)
    np.testing.assert_allclose(got_e, h + e / rms(e) * we, rtol=1e-13)


def test_linear_approximator_is_a_token_conditioned_bias():
    # Sec. 4 characterises the linear variant as a token-dependent offset added to the hidden
    # state: h' - h - W_lin^h h~ depends on the previous token alone (W_lin^e e), whatever the
    # hidden state, so rows of one depth differ by their tokens' offsets.
    H, root, W = small_problem(seed=8, gamma=3)
    d = H.shape[1]
    W["w_lin"] = np.random.default_rng(10).normal(0, 0.3, (d, 2 * d))
    _, ids, _ = O.stage1(H, W["lm_head"], 1.0, 4)
    hp, lp = O.stage2(H, root, ids, W, 3, 1.0, 1e-6, approx="linear")
    hid, prev = O.stage2_conditioning(3, 3, root, ids)
    h_part = O.rmsnorm(H[hid], W["norm_h"], 1e-6) @ W["w_lin"][:, :d].T
    bias = hp - H[hid] - h_part
    e_part = O.rmsnorm(W["embed"][prev], W["norm_e"], 1e-6) @ W["w_lin"][:, d:].T
    np.testing.assert_allclose(bias, e_part, atol=1e-12)
    # rows of one depth share h, so they differ by their tokens' embedding terms alone
    for a, b in ((1, 2), (2, 3), (4, 6)):
        np.testing.assert_allclose(hp[a] - hp[b], e_part[a] - e_part[b], atol=1e-12)
    np.testing.assert_allclose(np.exp(lp).sum(1), 1.0, rtol=1e-13)


def test_zero_linear_approximator_reduces_to_marginal_tree():
    # W_lin = 0 gives h' = h, so the linear variant's tree is the M-ary marginal tree
    for seed in range(3):
        H, root, W = small_problem(V=32, gamma=4, seed=seed)
        W["w_lin"] = np.zeros((H.shape[1], 2 * H.shape[1]))
        a = O.draft_sequence(H, root, 1000, W, M=3, K2=10, B=10, approx="linear")
        b = O.draft_sequence(H, root, 1000, W, M=3, K2=10, B=10, mode="marginal_mary")
        hid, _ = O.stage2_conditioning(4, 3, root, a.top_ids)
        np.testing.assert_array_equal(a.h_prime, H[hid])
        np.testing.assert_array_equal(a.tree.tok, b.tree.tok)
        np.testing.assert_array_equal(a.tree.parent, b.tree.parent)
        np.testing.assert_allclose(a.tree.score, b.tree.score, atol=1e-12)


# ------------------------------------------------------------------ Part 2: tree search


def _run(mode="ar", V=32, gamma=4, M=3, K2=None, B=10, seed=0, zero_wd=False, keep=None,
         literal=False, **kw):
    H, root, W = small_problem(V=V, gamma=gamma, seed=seed, **kw)
    if zero_wd:
        W["w_down"][:] = 0.0
    K2 = K2 if K2 is not None else B
    return O.draft_sequence(H, root, 1000, W, M=M, K2=K2, B=B, mode=mode, keep=keep,
                            literal=literal)


def _check_structure(res, B, gamma, M, mode):
    t = res.tree
    assert t.tok.shape == (B + 1,)
    assert t.parent[0] == -1 and t.depth[0] == 0 and t.score[0] == 0.0
    n = int((t.parent[1:] >= 0).sum()) + 1
    assert n == B + 1 and not t.underfull
    seen = set()
    for i in range(1, B + 1):
        p = t.parent[i]
        assert 0 <= p < i                                   # parent precedes child
        assert t.depth[i] == t.depth[p] + 1 <= gamma       # prefix-closed, depth cap
        assert t.score[i] <= t.score[p] + 1e-12             # monotone along paths
        key = (int(p), int(t.tok[i]))
        assert key not in seen                              # no duplicate children
        seen.add(key)
    scores = [s for s, *_ in t.pops]
    assert all(a >= b - 1e-12 for a, b in zip(scores, scores[1:]))   # pop order
    # non-leaf nodes lie in the M-ary tree (Sec. 3): their token is a stage-1 top-M
    if mode in ("ar", "marginal_mary"):
        for i in range(1, B + 1):
            if (t.parent == i).any():
                assert t.tok[i] in res.top_ids[t.depth[i] - 1, :M]
    # each score is the sum of log-probs along the path (OPT-Tree key, Sec. 3)
    for i in range(1, B + 1):
        p = t.parent[i]
        lp = res.s2_logp[t.row[i]] if mode == "ar" else res.s1_logp[t.row[i]]
        assert abs(t.score[i] - (t.score[p] + lp[t.tok[i]])) < 1e-12


@pytest.mark.parametrize("mode", ["ar", "marginal", "marginal_mary"])
@pytest.mark.parametrize("seed", [0, 1, 2])
def test_tree_structure_invariants(mode, seed):
    res = _run(mode=mode, seed=seed, B=14, M=3, gamma=4)
    _check_structure(res, 14, 4, 3, mode)


@pytest.mark.parametrize("mode", ["ar", "marginal", "marginal_mary"])
@pytest.mark.parametrize("keep", [None, 3])
def test_lazy_queue_equals_literal_algorithm(mode, keep):
    # Algorithm 1 Part 2 pushes whole distributions; the lazy queue must pick the same nodes
    for seed in range(4):
        a = _run(mode=mode, seed=seed, B=12, keep=keep, literal=True)
        b = _run(mode=mode, seed=seed, B=12, keep=keep, literal=False)
        for f in ("tok", "parent", "depth", "row"):
            np.testing.assert_array_equal(getattr(a.tree, f), getattr(b.tree, f))
        np.testing.assert_array_equal(a.tree.score, b.tree.score)


def test_lazy_equals_literal_with_exact_ties():
    # quantised weights make many exactly equal log-probs and path scores
    for seed in range(3):
        H, root, W = small_problem(V=12, gamma=3, seed=seed)
        for k in W:
            W[k] = np.round(W[k] * 2) / 2
        H = np.round(H)
        a = O.draft_sequence(H, root, 0, W, M=2, K2=9, B=9, literal=True)
        b = O.draft_sequence(H, root, 0, W, M=2, K2=9, B=9, literal=False)
        np.testing.assert_array_equal(a.tree.tok, b.tree.tok)
        np.testing.assert_array_equal(a.tree.parent, b.tree.parent)


def test_zeroed_approximator_reduces_to_marginal_tree():
    # W_down = 0 => q' = q for every row, so TreeFlash equals OPT-Tree on the marginals under
    # the M-ary rule; with M >= B - 1 the rule never binds and it equals DDTree.
    for seed in range(4):
        a = _run(mode="ar", seed=seed, zero_wd=True, B=10, M=3)
        b = _run(mode="marginal_mary", seed=seed, B=10, M=3)
        np.testing.assert_array_equal(a.tree.tok, b.tree.tok)
        np.testing.assert_array_equal(a.tree.parent, b.tree.parent)
        np.testing.assert_allclose(a.tree.score, b.tree.score, atol=1e-12)
        c = _run(mode="ar", seed=seed, zero_wd=True, B=6, M=5)
        e = _run(mode="marginal", seed=seed, B=6, M=5)
        np.testing.assert_array_equal(c.tree.tok, e.tree.tok)
        np.testing.assert_array_equal(c.tree.parent, e.tree.parent)


def _subtree_paths(t, node):
    kids = {}
    for i in range(1, t.tok.shape[0]):
        kids.setdefault(int(t.parent[i]), []).append(i)
    out = set()

    def walk(n, path):
        for c in kids.get(n, []):
            p = path + (int(t.tok[c]),)
            out.add(p)
            walk(c, p)
    walk(node, ())
    return out


def _is_nested(res):
    # App. C: for siblings a, b with q(a) > q(b) the subtree under b is contained in the
    # subtree under a (all siblings share one child ranking)
    t = res.tree
    for p in set(t.parent[1:].tolist()):
        sib = [i for i in range(1, t.tok.shape[0]) if t.parent[i] == p]
        sib.sort(key=lambda i: -t.score[i])
        for a, b in zip(sib, sib[1:]):
            if not _subtree_paths(t, b) <= _subtree_paths(t, a):
                return False
    return True


def test_marginal_trees_are_nested_and_ar_trees_need_not_be():
    assert all(_is_nested(_run(mode="marginal", seed=s, B=20, M=4)) for s in range(6))
    assert all(_is_nested(_run(mode="ar", seed=s, zero_wd=True, B=20, M=19)) for s in range(3))
    # with a strong approximator the child ranking depends on the previous token
    flags = [_is_nested(_run(mode="ar", seed=s, B=20, M=4, wd_std=3.0)) for s in range(6)]
    assert not all(flags)


def test_brute_force_top_b_of_eligible_universe():
    # V=16, gamma=4, M=4, B=12: enumerate every node the M-ary rule allows and confirm that
    # the tree is exactly the B best path scores (the greedy OPT-Tree optimum)
    for mode in ("ar", "marginal", "marginal_mary"):
        H, root, W = small_problem(V=16, d=16, gamma=4, seed=11, h_scale=2.0)
        res = O.draft_sequence(H, root, 0, W, M=4, K2=12, B=12, mode=mode)
        src = O.ChildSource(mode, 4, 4, res.top_ids, res.s1_logp, res.s2_logp)
        uni = O.eligible_universe(src)
        uni.sort(key=lambda x: (-x[0], x[1]))
        best = {p for _, _, p in uni[:12]}
        assert best == set(O.tree_paths(res.tree))
        assert uni[11][0] - uni[12][0] > 1e-9            # the comparison is not a tie


@pytest.mark.parametrize("mode", ["ar", "marginal"])
@pytest.mark.parametrize("B", [3, 5])
def test_exhaustive_prefix_closed_optimum(mode, B):
    # V=4, gamma=3: search all prefix-closed sets of B nodes for the largest summed path
    # probability (expected accepted tokens, Sec. 3); the selected tree attains it
    H, root, W = small_problem(V=4, d=8, I=8, gamma=3, seed=13, h_scale=1.5)
    res = O.draft_sequence(H, root, 0, W, M=2, K2=B, B=B, mode=mode)
    src = O.ChildSource(mode, 3, 2, res.top_ids, res.s1_logp, res.s2_logp)
    uni = O.eligible_universe(src)
    got = sum(math.exp(s) for s in res.tree.score[1:])
    assert abs(O.best_prefix_closed_value(uni, B) - got) < 1e-12


def test_budget_truncation_k2_less_than_b():
    # reading R5: K2 >= B is exact; K2 < B keeps at most K2 children per distribution
    exact = _run(seed=3, B=12, K2=12)
    full = _run(seed=3, B=12, keep=None)
    np.testing.assert_array_equal(exact.tree.tok, full.tree.tok)
    t = _run(seed=3, B=12, K2=2, keep=2).tree
    for p in set(t.parent[1:].tolist()):
        rows = {}
        for i in range(1, 13):
            if t.parent[i] == p:
                rows.setdefault(t.row[i], []).append(i)
        assert all(len(v) <= 2 for v in rows.values())


def test_underfull_universe_is_flagged():
    # gamma = 1 and K2 = 3 children at the root: only 3 nodes exist for B = 5
    H, root, W = small_problem(V=8, gamma=1, seed=1)
    res = O.draft_sequence(H, root, 0, W, M=2, K2=3, B=5, keep=3)
    assert res.tree.underfull
    assert list(res.tree.parent[4:]) == [-1, -1]
    assert res.pos[4] == -1 and res.mask[4].sum() == 0 and res.mask[:, 4].sum() == 0


def test_hand_worked_tree():
    # Probabilities are powers of two, so sums of their logs are exact and the tie below is
    # a true tie. DDTree (marginals), gamma = 2, V = 4, B = 3:
    #   depth 1: p = (1/2, 1/4, 1/8, 1/8), depth 2: the same.
    # queue after the root: t0:1/2, t1:1/4, t2:1/8, t3:1/8      -> pop t0 (node 1)
    # push node 1's children: (t0,t0):1/4, (t0,t1):1/8, ...
    # t1 (depth 1) and (t0,t0) (depth 2) tie at 1/4: the smaller depth wins -> pop t1 (node 2)
    # then (t0,t0):1/4 beats everything else                    -> pop it (node 3)
    d1 = np.log([0.5, 0.25, 0.125, 0.125])
    src = O.ChildSource("marginal", 2, 1, np.array([[0, 1, 2, 3], [0, 1, 2, 3]]),
                        np.stack([d1, d1]), None)
    t = O.build_tree_literal(src, root_tok=9, B=3)
    assert list(t.tok) == [9, 0, 1, 0]
    assert list(t.parent) == [-1, 0, 0, 1]
    assert list(t.depth) == [0, 1, 1, 2]
    np.testing.assert_array_equal(np.exp(t.score[1:]), [0.5, 0.25, 0.25])
    # TreeFlash, M = 2, stage-1 depth-1 candidates (t1, t0): t0 is candidate m = 1, so its
    # children come from stage-2 row 1 + (1 - 1) * 2 + 1 = 2; t1 (m = 0) uses row 1.
    #   row 0 (root's children): (1/2, 1/4, 1/8, 1/8)
    #   row 1: (1/2, 1/4, 1/8, 1/8); row 2: (1/8, 1/8, 1/2, 1/4)
    # pop t0 (1/2); push (t0,t2) = 1/4; t1 ties with it at 1/4 and wins on depth -> pop t1;
    # push (t1,t0) = 1/8; then (t0,t2) = 1/4 is popped.
    s2 = np.log(np.array([[0.5, 0.25, 0.125, 0.125], [0.5, 0.25, 0.125, 0.125],
                          [0.125, 0.125, 0.5, 0.25]]))
    src = O.ChildSource("ar", 2, 2, np.array([[1, 0, 2, 3], [0, 1, 2, 3]]),
                        np.stack([d1, d1]), s2)
    t = O.build_tree_literal(src, root_tok=9, B=3)
    assert list(t.tok) == [9, 0, 1, 2]
    assert list(t.parent) == [-1, 0, 0, 1]
    assert list(t.row) == [-1, 0, 0, 2]
    np.testing.assert_array_equal(np.exp(t.score[1:]), [0.5, 0.25, 0.25])


# ------------------------------------------------------------------ mask


@pytest.mark.parametrize("mode", ["ar", "marginal"])
def test_mask_invariants(mode):
    res = _run(mode=mode, seed=4, B=16, M=4)
    m = res.mask.astype(np.int64)
    n = m.shape[0]
    assert (np.diag(m) == 1).all()
    # the ancestor relation is transitive: (m @ m > 0) == m
    np.testing.assert_array_equal((m @ m > 0).astype(np.int64), m)
    np.testing.assert_array_equal(m.sum(1), res.tree.depth + 1)
    assert (np.triu(m, 1) == 0).all()          # ancestors precede descendants
    for i in range(1, n):
        assert m[i, res.tree.parent[i]] == 1
    np.testing.assert_array_equal(res.pos, 1000 + res.tree.depth)


def test_topk_margin_hand_values():
    # the gap between the k-th and (k+1)-th largest entries, by hand; every value is a binary
    # fraction, so the differences are exact
    v = np.array([5.0, 1.0, 3.0, 2.5, -1.0])
    assert [O.topk_margin(v, k) for k in (1, 2, 3, 4)] == [2.0, 0.5, 1.5, 2.0]
    assert O.topk_margin(v, 5) == np.inf


def _hand_result(mode, s1, s2, M, K2, B):
    """A SeqResult built from hand-written (unnormalised) log-probability lists; ids ranked
    by value, the tree by the lazy builder."""
    s1 = np.array(s1, dtype=np.float64)
    s2 = None if s2 is None else np.array(s2, dtype=np.float64)
    top_ids = np.stack([O.ranked(r, s1.shape[1]) for r in s1])
    src = O.ChildSource(mode, s1.shape[0], M, top_ids, s1, s2)
    tree = O.build_tree_lazy(src, 9, B, keep=K2 if K2 < B else None)
    return O.SeqResult(s1, top_ids, None, None, s2, None, None, tree, None, None)


def test_selection_margins_hand_values():
    # The margins that decide where the GPU tree must match exactly, on hand-made lists whose
    # gaps are known exactly. A wrong rank (k vs k + 1), a wrong (B+1)-th pop or a missing term
    # changes at least one of the expected values below.
    #
    # DDTree (marginal), gamma = 2, B = 2. Universe: t0 -1, (t0,u0) -1.25, t1 -2.25,
    # (t1,u0) -2.5, ... Pops: -1, -1.25; the best left out is t1 at -2.25, so the set margin
    # is 1.0 and the order margin (gap between the two pops) 0.25. The stage-1 rank-M gap
    # (0.0625 at M = 2) does not enter: DDTree expands every node.
    r = _hand_result("marginal", [[-1, -2.25, -2.3125, -7], [-0.25, -3, -3.5, -9]], None, M=2, K2=4, B=2)
    assert list(r.tree.tok) == [9, 0, 0]
    assert O.selection_margins(r, 2, 4, 2, "marginal") == (1.0, 0.25)
    # TreeFlash, gamma = 2, M = 2: stage-2 row 0 holds the root's children, row 1 the children
    # of depth-1 candidate 0 (token 0), row 2 those of candidate 1 (token 1).
    s2 = [[-0.5, -2, -2.5, -6], [-1, -1.125, -4, -4.5], [-0.375, -3, -3.125, -4]]
    # Rank-M gap of depth 1: 3.0. Universe: t0 -0.5, (t0,0) -1.5, (t0,1) -1.625, t1 -2,
    # (t1,0) -2.375, t2 -2.5, ... (t2, t3 are leaves). B = 3 pops -0.5, -1.5, -1.625; the best
    # left out is t1 at -2, so the set margin is min(3.0, 0.375) and the order margin
    # min(0.375, 1.0, 0.125).
    wide = [[-1, -1.5, -4.5, -5], [-1, -2, -3, -4]]
    r = _hand_result("ar", wide, s2, M=2, K2=4, B=3)
    assert list(r.tree.tok) == [9, 0, 0, 1]
    assert O.selection_margins(r, 2, 4, 3, "ar") == (0.375, 0.125)
    # the same with the stage-1 rank-M gap of depth 1 shrunk to 0.125: it decides both
    narrow = [[-1, -1.5, -1.625, -5], [-1, -2, -3, -4]]
    r = _hand_result("ar", narrow, s2, M=2, K2=4, B=3)
    assert O.selection_margins(r, 2, 4, 3, "ar") == (0.125, 0.125)
    # K2 = 2 < B = 3 truncates every list after two entries; the rank-2 gaps of the stage-2
    # rows are 0.5, 2.875 and 0.125 (row 2), the smallest term of the set margin
    r = _hand_result("ar", wide, s2, M=2, K2=2, B=3)
    assert list(r.tree.tok) == [9, 0, 0, 1]
    assert O.selection_margins(r, 2, 2, 3, "ar") == (0.125, 0.125)


def test_margins_are_positive_and_finite_for_generic_inputs():
    res = _run(seed=5, B=10, M=3)
    sm, om = O.selection_margins(res, 3, 10, 10)
    assert 0 < om <= sm < np.inf


def test_oracle_matches_frozen_golden():
    # regression guard: tests/golden/tiny_f32_seed0.json was written by
    # tests/golden/make_golden.py (oracle + synth only)
    import json
    import os
    import synth
    path = os.path.join(os.path.dirname(__file__), "golden", "tiny_f32_seed0.json")
    gold = json.load(open(path))
    for name, g in gold.items():
        cfg = synth.get_config(name)
        inp = synth.make_inputs(cfg)
        W = O.weights_f64(inp, synth.to_f64)
        res = O.draft_sequence(synth.to_f64(inp["hidden"])[0], int(inp["root_tok"][0]),
                               int(inp["root_pos"][0]), W, M=cfg.M, K2=cfg.K2, B=cfg.B)
        assert res.tree.tok.tolist() == g["tok"]
        assert res.tree.parent.tolist() == g["parent"]
        np.testing.assert_allclose(res.tree.score, g["score"], rtol=1e-12)


def test_oracle_variants_match_frozen_golden():
    # the same guard for the ablations' approximators (tests/golden/tiny_variants_seed0.json)
    import json
    import os
    import synth
    path = os.path.join(os.path.dirname(__file__), "golden", "tiny_variants_seed0.json")
    gold = json.load(open(path))
    assert set(gold) == {"tiny_peaked/linear", "tiny_peaked/swiglu_2prev"}
    for key, g in gold.items():
        name, approx = key.split("/")
        cfg = synth.get_config(name, approx=approx)
        inp = synth.make_inputs(cfg)
        W = O.weights_f64(inp, synth.to_f64)
        prev = int(inp["root_prev"][0]) if "root_prev" in inp else None
        res = O.draft_sequence(synth.to_f64(inp["hidden"])[0], int(inp["root_tok"][0]),
                               int(inp["root_pos"][0]), W, M=cfg.M, K2=cfg.K2, B=cfg.B, approx=approx,
                               root_prev=prev)
        assert res.tree.tok.tolist() == g["tok"]
        assert res.tree.parent.tolist() == g["parent"]
        np.testing.assert_allclose(res.tree.score, g["score"], rtol=1e-12)
        np.testing.assert_allclose(res.child_logp[0], g["child_logp_row0"], rtol=1e-12)


# ------------------------------------------------------------------ verification walk


def test_accept_walk_hand_worked():
    # root 0 -> 1 (5), 2 (7); 1 -> 3 (9), 4 (11); 3 -> 5 (2); node 6 missing
    tok = np.array([100, 5, 7, 9, 11, 2, -1])
    par = np.array([-1, 0, 0, 1, 1, 3, -1])
    # the verifier continues 5, 9, 2 and then proposes 42: three drafted tokens accepted, tau 4
    path, bonus = O.accept_walk(tok, par, np.array([5, 9, 0, 2, 0, 42, 0]))
    assert path == [0, 1, 3, 5] and bonus == 42
    # the verifier's first token is not drafted: nothing accepted, the step gains one token
    path, bonus = O.accept_walk(tok, par, np.array([8, 9, 0, 2, 0, 42, 0]))
    assert path == [0] and bonus == 8
    # the second branch, stopping where no child matches (node 4 has none)
    path, bonus = O.accept_walk(tok, par, np.array([5, 11, 0, 2, 17, 42, 0]))
    assert path == [0, 1, 4] and bonus == 17
    # a missing node is never accepted, even if its token matches
    path, _ = O.accept_walk(tok, par, np.array([7, 0, -1, 0, 0, 0, 0]))
    assert path == [0, 2]


def _node_paths(par):
    # every root path, as node indices, by walking parent links from each node
    out = []
    for i in range(len(par)):
        if i > 0 and par[i] < 0:
            continue
        p, j = [], i
        while j > 0:
            p.append(j)
            j = int(par[j])
        out.append([0] + p[::-1])
    return out


@pytest.mark.parametrize("seed", range(6))
def test_accept_walk_is_the_longest_consistent_root_path(seed):
    # brute force over all root paths of an oracle tree: the accepted path is the longest path
    # along which every drafted token equals the verifier's token at its parent, and the bonus
    # is the verifier's token at its end
    res = _run(seed=seed, B=12, M=3)
    tok, par = res.tree.tok, res.tree.parent
    n = len(tok)
    rng = np.random.default_rng(100 + seed)
    children = {i: [c for c in range(1, n) if par[c] == i] for i in range(n)}
    ver = np.empty(n, dtype=np.int64)
    for i in range(n):
        if children[i] and rng.random() < 0.7:
            ver[i] = tok[rng.choice(children[i])]    # the verifier agrees with one child
        else:
            ver[i] = 10_000 + i                      # a token no node carries
    consistent = [p for p in _node_paths(par) if all(tok[b] == ver[a] for a, b in zip(p, p[1:]))]
    best = max(consistent, key=len)
    assert sum(1 for p in consistent if len(p) == len(best)) == 1
    path, bonus = O.accept_walk(tok, par, ver)
    assert path == best and bonus == ver[best[-1]]
    assert 1 <= len(path) <= res.tree.depth.max() + 1


# ------------------------------------------------------------------ "w/ 2-prev" approximator
# (Sec. 4 "Model Design", Table 3; reading R13): x = [h~ ; e(prev) ; e(token before prev)],
# one stage-2 row per pair of M-ary candidates of the two previous depths.


def small_problem_2prev(V=32, d=16, I=24, gamma=4, seed=0, extra_std=0.3, **kw):
    """small_problem with gate/up widened to [I, 3d] (extra columns for the second previous
    token) and a token before the root."""
    H, root, W = small_problem(V=V, d=d, I=I, gamma=gamma, seed=seed, **kw)
    rng = np.random.default_rng(1000 + seed)
    W = dict(W, w_gate=np.hstack([W["w_gate"], rng.normal(0, extra_std, (I, d))]),
             w_up=np.hstack([W["w_up"], rng.normal(0, extra_std, (I, d))]))
    return H, root, int(rng.integers(0, V)), W


def test_2prev_row_layout():
    # gamma = 3, M = 2: depth 1 on (root, token before it); depth 2 on (candidate m of depth 1,
    # root); depth 3 on (candidate m1 of depth 2, candidate m2 of depth 1), m1-major
    top = np.array([[10, 11, 99], [20, 21, 98], [30, 31, 97]])
    hid, p1, p2 = O.stage2_conditioning_2prev(3, 2, root_tok=7, root_prev=5, top_ids=top)
    assert hid.tolist() == [0, 1, 1, 2, 2, 2, 2]
    assert p1.tolist() == [7, 10, 11, 20, 20, 21, 21]
    assert p2.tolist() == [5, 7, 7, 10, 11, 10, 11]
    assert O.stage2_rows(3, 2, "swiglu_2prev") == 7 == len(hid)
    assert O.stage2_rows(16, 16, "swiglu_2prev") == 1 + 16 + 256 * 14
    assert O.stage2_rows(1, 16, "swiglu_2prev") == 1
    # the child row of a node is the row conditioned on (its token, its parent's token)
    src = O.ChildSource("ar", 3, 2, top, np.zeros((3, 4)), np.zeros((7, 4)), approx="swiglu_2prev")
    assert src.child_row(1, 11, 7) == 2
    assert [src.child_row(2, t, pt) for t in (20, 21) for pt in (10, 11)] == [3, 4, 5, 6]
    for r in range(3, 7):
        assert (p1[r], p2[r]) == ({3: 20, 4: 20, 5: 21, 6: 21}[r], {3: 10, 4: 11, 5: 10, 6: 11}[r])
    assert src.child_row(2, 99, 10) is None and src.child_row(3, 30, 20) is None


def test_2prev_approximator_hand_computed():
    # d = 2, I = 1, norm weights 1, eps = 0; h = (3, 4), e = (1, -1), e2 = (2, 0): RMS sqrt(2)
    h, e, e2 = np.array([[3.0, 4.0]]), np.array([[1.0, -1.0]]), np.array([[2.0, 0.0]])
    wg = np.array([[1.0, 0.0, 0.0, 0.0, 1.0, 0.0]])    # G = x0 + x4
    wu = np.array([[0.0, 1.0, 0.0, 0.0, 0.0, -1.0]])   # U = x1 - x5
    wd = np.array([[2.0], [-1.0]])
    x0, x1, x4, x5 = 3 / math.sqrt(12.5), 4 / math.sqrt(12.5), 2 / math.sqrt(2), 0.0
    G, U = x0 + x4, x1 - x5
    a = G / (1 + math.exp(-G)) * U
    got = O.ar_approximator(h, e, np.ones(2), np.ones(2), wg, wu, wd, 0.0, e2_raw=e2)
    np.testing.assert_allclose(got, np.array([[3 + 2 * a, 4 - a]]), rtol=1e-14)


def _run_2prev(zero_extra=False, approx="swiglu_2prev", V=32, gamma=4, M=3, B=12, seed=0, literal=False,
               **kw):
    H, root, prev, W = small_problem_2prev(V=V, gamma=gamma, seed=seed, **kw)
    d = H.shape[1]
    if zero_extra:
        W["w_gate"][:, 2 * d:] = 0.0
        W["w_up"][:, 2 * d:] = 0.0
    if approx == "swiglu":
        W = dict(W, w_gate=W["w_gate"][:, :2 * d], w_up=W["w_up"][:, :2 * d])
    return O.draft_sequence(H, root, 1000, W, M=M, K2=B, B=B, approx=approx, root_prev=prev,
                            literal=literal)


def test_2prev_without_second_token_columns_equals_treeflash():
    # zero columns for the second previous token: every row (i, m1, m2) is TreeFlash's row
    # (i, m1), so the trees coincide (pins the row layout and the child-row rule together)
    for seed in range(4):
        a = _run_2prev(zero_extra=True, seed=seed)
        b = _run_2prev(approx="swiglu", seed=seed)
        M, g = 3, 4
        for r in range(O.stage2_rows(g, M, "swiglu_2prev")):
            if r == 0:
                rb = 0
            elif r <= M:
                rb = r
            else:
                q = r - 1 - M
                rb = 1 + (2 + q // (M * M) - 1) * M + (q % (M * M)) // M
            np.testing.assert_allclose(a.s2_logp[r], b.s2_logp[rb], atol=1e-12)
        np.testing.assert_array_equal(a.tree.tok, b.tree.tok)
        np.testing.assert_array_equal(a.tree.parent, b.tree.parent)
        np.testing.assert_allclose(a.tree.score, b.tree.score, atol=1e-12)


def test_2prev_second_token_matters():
    # with non-zero columns the rows of one (depth, previous token) differ by the token before
    a = _run_2prev(seed=2, extra_std=1.0)
    M = 3
    r = 1 + M                       # depth 3, candidates (m1 = 0, m2 = 0) and (0, 1)
    assert np.abs(a.s2_logp[r] - a.s2_logp[r + 1]).max() > 1e-3


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_2prev_tree_invariants_and_literal(seed):
    res = _run_2prev(seed=seed, B=14, h_scale=2.0, extra_std=1.0)
    _check_structure(res, 14, 4, 3, "ar")
    t = res.tree
    # every node's list is the row of (its parent's token, its grandparent's token)
    for i in range(1, 15):
        p = int(t.parent[i])
        if t.depth[i] == 1:
            assert t.row[i] == 0
        elif t.depth[i] == 2:
            assert t.row[i] == 1 + res.top_ids[0, :3].tolist().index(t.tok[p])
        else:
            gp = int(t.parent[p])
            dp = int(t.depth[p])
            m = res.top_ids[dp - 1, :3].tolist().index(t.tok[p])
            mp = res.top_ids[dp - 2, :3].tolist().index(t.tok[gp])
            assert t.row[i] == 1 + 3 + (dp - 2) * 9 + m * 3 + mp
    lit = _run_2prev(seed=seed, B=14, h_scale=2.0, extra_std=1.0, literal=True)
    np.testing.assert_array_equal(lit.tree.tok, t.tok)
    np.testing.assert_array_equal(lit.tree.parent, t.parent)


def test_2prev_brute_force_top_b_and_exhaustive_optimum():
    # V = 16: the tree is the B best path scores of every node the rule allows; V = 4: it
    # attains the largest summed path probability over all prefix-closed sets
    H, root, prev, W = small_problem_2prev(V=16, d=16, gamma=4, seed=11, h_scale=2.0, extra_std=1.0)
    res = O.draft_sequence(H, root, 0, W, M=4, K2=12, B=12, approx="swiglu_2prev", root_prev=prev)
    src = O.ChildSource("ar", 4, 4, res.top_ids, res.s1_logp, res.s2_logp, approx="swiglu_2prev")
    uni = O.eligible_universe(src)
    uni.sort(key=lambda x: (-x[0], x[1]))
    assert {p for _, _, p in uni[:12]} == set(O.tree_paths(res.tree))
    assert uni[11][0] - uni[12][0] > 1e-9
    H, root, prev, W = small_problem_2prev(V=4, d=8, I=8, gamma=3, seed=13, h_scale=1.5, extra_std=1.0)
    for B in (3, 5):
        res = O.draft_sequence(H, root, 0, W, M=2, K2=B, B=B, approx="swiglu_2prev", root_prev=prev)
        src = O.ChildSource("ar", 3, 2, res.top_ids, res.s1_logp, res.s2_logp, approx="swiglu_2prev")
        got = sum(math.exp(s) for s in res.tree.score[1:])
        assert abs(O.best_prefix_closed_value(O.eligible_universe(src), B) - got) < 1e-12
