"""TreeFlash drafting path: plain fp64 CPU oracle.

TEST INFRASTRUCTURE ONLY. Only tests/, __graft_entry__.smoke() and bench.py (its
cpu_baseline leg and its reference arm) may import this module. The product path (the
CUDA library and its Python binding) never imports, links or executes it, and this module
imports nothing from the product package.

What it computes (TreeFlash, "Parallel AR-Approximation for Faster Speculative Decoding"):

* Part 1 of the AR-approximated OPT-Tree construction (Algorithm 1 in App. B):
  - stage 1: for every depth i, the marginal q_{t+i} = LMHead(h_{t+i}) and its top-M
    candidates x^(1..M)_{t+i};
  - stage 2: the AR-approximator of Eq. 1, h' = h + SwiGLU(h~ :: e), evaluated on one row
    for depth 1 (conditioned on the root token x_t) and on M rows for every depth
    i = 2..gamma (conditioned on the stage-1 candidates of depth i-1), each projected
    through the LM head into q'; optionally with the "w/ Linear" ablation's linear layer in
    place of the SwiGLU (reading R12).
* Part 2 of Algorithm 1: OPT-Tree best-first selection (Sec. 3, "Inference") of B nodes by
  cumulative path log-probability; a popped node at depth i whose token is the stage-1
  candidate m of depth i gets the children distribution q'^(m)_{t+i+1}.
* The verifier's tree-attention mask and position ids for the B+1 nodes (the tree is
  verified in one parallel forward pass, Sec. 1 and Sec. 3).
* The verification walk over a drafted tree: acceptance by an equality check with the
  verifier's tokens (Sec. 3) and the step's block efficiency tau (Sec. 4).

Everything is float64 (numpy). Library primitives used as steps: matrix products, sorting,
exp/log. Readings of points the paper leaves open (each also listed in the design notes):

  R1  "normalized" hidden state / input embedding (Eq. 1): RMSNorm with a learnable weight,
      y = x / sqrt(mean(x^2) + eps) * w, eps = 1e-6 (the Qwen3 verifier family's norm).
  R2  LMHead(x) = W_lm x / T: the verifier's output embedding with no final norm, T = 1.
  R3  SwiGLU(x) = W_down (SiLU(W_gate x) * (W_up x)), x = [h~ ; e] in R^{2d} (h~ first).
  R4  Stage-2 row count: Algorithm 1 gives 1 + M (gamma - 1) rows (row 0: depth 1 from
      the root; row 1 + (i-2) M + m: depth i, candidate m of depth i-1).
  R5  Queue contents: Algorithm 1 pushes a whole distribution. Keeping the top K2 >= B
      children of each row is exactly equivalent; K2 < B truncates (modelled by `keep`).
  R6  Budget: B excludes the root; the tree has B + 1 entries, node 0 the root.
  R7  Depth cap: nodes at depth gamma are never expanded.
  R8  Ties (the paper is silent): inside a distribution, larger value first, then smaller
      token id. In the queue: larger score, then smaller depth, then smaller parent index
      (pop order), then smaller token id. Nodes are numbered in pop order.
  R9  If fewer than B candidates exist, the tree holds what exists and is flagged.
  R10 Marginal baselines: "marginal" is DDTree (OPT-Tree on the stage-1 marginals, every
      node expandable, Sec. 4 "Baselines"); "marginal_mary" is the same search restricted
      by the M-ary rule of Sec. 3 (what TreeFlash reduces to with a zeroed approximator).
  R12 The "w/ Linear" ablation (Sec. 4 "Model Design", Table 3) replaces the SwiGLU of
      Eq. 1 by one linear map on the same input: h' = h + W_lin (h~ :: e), W_lin [d, 2d],
      no bias vector. The token-dependent part of h' is then W_lin's embedding half applied
      to e, the same for every hidden state: the token-dependent offset of the hidden state
      that Sec. 4 attributes to this variant.
  R13 The "w/ 2-prev" ablation (Sec. 4 "Model Design", Table 3) conditions on the two
      previous tokens: x = [h~ ; e(x_{t+i-1}) ; e(x_{t+i-2})] in R^{3d} (both embeddings
      normalised with the one input-embedding norm weight), W_gate, W_up [I, 3d]. Depth 1
      conditions on (x_t, x_{t-1}), so the step also takes the token before the root. The
      M-ary tree then needs one row per pair of candidates: row 0 for depth 1, rows 1..M
      for depth 2 (candidate m of depth 1, x_t), and row 1 + M + (i-3) M^2 + m1 M + m2 for
      depth i >= 3 (candidate m1 of depth i-1, candidate m2 of depth i-2): 1 + M + M^2
      (gamma - 2) rows. A popped node of depth i whose token is candidate m of depth i and
      whose parent's token is candidate m' of depth i-1 gets the children of row
      (i+1, m, m'); its parent is in the M-ary tree because it was expanded.

Optional bf16 emulation (`emulate_bf16=True`) rounds to bfloat16 (round to nearest even)
exactly where a bf16 implementation stores intermediates: the RMSNorm outputs, SiLU(G)*U,
and h'. With it off this is the plain fp64 definition.
"""
from __future__ import annotations

import heapq
import itertools
from dataclasses import dataclass, field
from typing import List, Optional, Sequence

import numpy as np

NEG_INF = -np.inf

# ---------------------------------------------------------------------------------------
# elementary pieces
# ---------------------------------------------------------------------------------------


def bf16_round(x: np.ndarray) -> np.ndarray:
    """Round float64 values to the nearest bfloat16 value (ties to even), returned as
    float64. bfloat16 keeps 8 significant bits; frexp gives x = f * 2^e with 0.5 <= |f| < 1,
    so f * 2^8 is rounded to an integer (np.rint rounds half to even) and scaled back.
    Finite, normal-range inputs only (all this path produces)."""
    x = np.asarray(x, dtype=np.float64)
    f, e = np.frexp(x)
    return np.ldexp(np.rint(np.ldexp(f, 8)), e - 8)


def rmsnorm(x: np.ndarray, w: np.ndarray, eps: float) -> np.ndarray:
    """Reading R1 of the normalisation in Eq. 1: x / sqrt(mean(x^2) + eps) * w (last axis)."""
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return x / np.sqrt(ms + eps) * w


def silu(x: np.ndarray) -> np.ndarray:
    return x / (1.0 + np.exp(-x))


def lm_head(x: np.ndarray, W_lm: np.ndarray, temperature: float) -> np.ndarray:
    """LMHead of Algorithm 1 (reading R2): logits W_lm x / T for each row of x."""
    return (x @ W_lm.T) / temperature


def log_softmax(z: np.ndarray) -> np.ndarray:
    """log q = z - log sum_v exp(z_v), with the max shift, per row."""
    m = np.max(z, axis=-1, keepdims=True)
    return z - (m + np.log(np.sum(np.exp(z - m), axis=-1, keepdims=True)))


def ranked(values: np.ndarray, k: Optional[int] = None) -> np.ndarray:
    """Indices of `values` (1-D) in the order of reading R8: larger value first, equal
    values by smaller index. A stable sort of -values keeps equal keys in index order."""
    order = np.argsort(-values, kind="stable")
    return order if k is None else order[:k]


# ---------------------------------------------------------------------------------------
# Part 1 of Algorithm 1
# ---------------------------------------------------------------------------------------


def stage1(H: np.ndarray, W_lm: np.ndarray, temperature: float, K1: int):
    """Stage 1 for one sequence: H [gamma, d] -> (logp [gamma, V], top_ids [gamma, K1],
    top_logp [gamma, K1]). The first M entries of top_ids are x^(1..M) of Algorithm 1."""
    logp = log_softmax(lm_head(H, W_lm, temperature))
    ids = np.stack([ranked(row, K1) for row in logp])
    return logp, ids, np.take_along_axis(logp, ids, axis=1)


def stage2_conditioning(gamma: int, M: int, root_tok: int, top_ids: np.ndarray):
    """Reading R4: for each stage-2 row, (index of the hidden state it refines, previous
    token it is conditioned on). Row 0: depth 1 with the root token; row 1 + (i-2) M + m:
    depth i in 2..gamma with stage-1 candidate m of depth i-1."""
    hid = [0]
    prev = [int(root_tok)]
    for i in range(2, gamma + 1):
        for m in range(M):
            hid.append(i - 1)
            prev.append(int(top_ids[i - 2, m]))
    return np.array(hid, dtype=np.int64), np.array(prev, dtype=np.int64)


def ar_approximator(h: np.ndarray, e_raw: np.ndarray, norm_h: np.ndarray, norm_e: np.ndarray,
                    w_gate: np.ndarray, w_up: np.ndarray, w_down: np.ndarray, eps: float,
                    emulate_bf16: bool = False, e2_raw: Optional[np.ndarray] = None) -> np.ndarray:
    """Eq. 1 on a batch of rows: h' = h + SwiGLU(h~ :: e) with h~ = RMSNorm(h) * norm_h and
    e = RMSNorm(E[prev]) * norm_e (readings R1, R3). h, e_raw: [rows, d]. With e2_raw (the
    embeddings of the token before prev, reading R13) the input is h~ :: e :: e2."""
    rnd = bf16_round if emulate_bf16 else (lambda a: a)
    parts = [rnd(rmsnorm(h, norm_h, eps)), rnd(rmsnorm(e_raw, norm_e, eps))]
    if e2_raw is not None:
        parts.append(rnd(rmsnorm(e2_raw, norm_e, eps)))
    x = np.concatenate(parts, axis=1)
    a = rnd(silu(x @ w_gate.T) * (x @ w_up.T))
    return rnd(h + a @ w_down.T)


def linear_approximator(h: np.ndarray, e_raw: np.ndarray, norm_h: np.ndarray, norm_e: np.ndarray,
                        w_lin: np.ndarray, eps: float, emulate_bf16: bool = False) -> np.ndarray:
    """The "w/ Linear" ablation (reading R12): h' = h + W_lin (h~ :: e) with the same
    normalised input as Eq. 1. h, e_raw: [rows, d]; w_lin: [d, 2d]."""
    rnd = bf16_round if emulate_bf16 else (lambda a: a)
    x = np.concatenate([rnd(rmsnorm(h, norm_h, eps)), rnd(rmsnorm(e_raw, norm_e, eps))], axis=1)
    return rnd(h + x @ w_lin.T)


def stage2_rows(gamma: int, M: int, approx: str = "swiglu") -> int:
    """Stage-2 rows of one sequence (readings R4, R13)."""
    if approx == "swiglu_2prev":
        return 1 if gamma == 1 else 1 + M + M * M * (gamma - 2)
    return 1 + M * (gamma - 1)


def stage2_conditioning_2prev(gamma: int, M: int, root_tok: int, root_prev: int, top_ids: np.ndarray):
    """Reading R13: for each stage-2 row, (index of the hidden state it refines, previous
    token, the token before that)."""
    hid, p1, p2 = [0], [int(root_tok)], [int(root_prev)]
    if gamma >= 2:
        for m in range(M):
            hid.append(1)
            p1.append(int(top_ids[0, m]))
            p2.append(int(root_tok))
    for i in range(3, gamma + 1):
        for m1 in range(M):
            for m2 in range(M):
                hid.append(i - 1)
                p1.append(int(top_ids[i - 2, m1]))
                p2.append(int(top_ids[i - 3, m2]))
    return (np.array(hid, dtype=np.int64), np.array(p1, dtype=np.int64), np.array(p2, dtype=np.int64))


def stage2(H: np.ndarray, root_tok: int, top_ids: np.ndarray, W: dict, M: int,
           temperature: float, eps: float, emulate_bf16: bool = False, approx: str = "swiglu",
           root_prev: Optional[int] = None):
    """Stage 2 for one sequence: returns (h_prime [R, d], logp [R, V]). approx: "swiglu"
    (Eq. 1), "linear" (reading R12) or "swiglu_2prev" (reading R13, which also needs the
    token before the root, root_prev)."""
    gamma = H.shape[0]
    if approx == "swiglu_2prev":
        if root_prev is None:
            raise ValueError("the two-previous-token approximator needs root_prev")
        hid, p1, p2 = stage2_conditioning_2prev(gamma, M, root_tok, root_prev, top_ids)
        hp = ar_approximator(H[hid], W["embed"][p1], W["norm_h"], W["norm_e"], W["w_gate"], W["w_up"],
                             W["w_down"], eps, emulate_bf16, e2_raw=W["embed"][p2])
        return hp, log_softmax(lm_head(hp, W["lm_head"], temperature))
    hid, prev = stage2_conditioning(gamma, M, root_tok, top_ids)
    if approx == "swiglu":
        hp = ar_approximator(H[hid], W["embed"][prev], W["norm_h"], W["norm_e"],
                             W["w_gate"], W["w_up"], W["w_down"], eps, emulate_bf16)
    elif approx == "linear":
        hp = linear_approximator(H[hid], W["embed"][prev], W["norm_h"], W["norm_e"],
                                 W["w_lin"], eps, emulate_bf16)
    else:
        raise ValueError(approx)
    return hp, log_softmax(lm_head(hp, W["lm_head"], temperature))


# ---------------------------------------------------------------------------------------
# Part 2 of Algorithm 1: OPT-Tree best-first selection
# ---------------------------------------------------------------------------------------


@dataclass
class Tree:
    tok: np.ndarray       # [B+1] int64, node 0 = root token
    parent: np.ndarray    # [B+1] int64, -1 for the root (and for missing nodes)
    depth: np.ndarray     # [B+1] int64
    score: np.ndarray     # [B+1] float64: cumulative path log-probability (root 0)
    row: np.ndarray       # [B+1] int64: the distribution a node was drawn from (-1 root)
    underfull: bool = False
    pops: List[tuple] = field(default_factory=list)  # queue keys in pop order


class ChildSource:
    """Which distribution the children of a node come from (Algorithm 1 Part 2, the
    'if v = x^(m)_{t+i}' step, and reading R10 for the marginal baselines).

    rows: list of 1-D log-probability arrays (distributions); root_row: index of the
    distribution of the root's children; child_row(depth, tok, parent_tok) -> index or None
    (parent_tok, the token of the node's parent, matters only for reading R13)."""

    def __init__(self, mode: str, gamma: int, M: int, stage1_top_ids: np.ndarray,
                 stage1_logp: np.ndarray, stage2_logp: Optional[np.ndarray], approx: str = "swiglu"):
        self.mode, self.gamma, self.M = mode, gamma, M
        self.two_prev = mode == "ar" and approx == "swiglu_2prev"
        self.top_m = [list(map(int, stage1_top_ids[i, :M])) for i in range(gamma)]
        if mode == "ar":
            self.rows = list(stage2_logp)
            self.root_row = 0
        elif mode in ("marginal", "marginal_mary"):
            self.rows = list(stage1_logp)
            self.root_row = 0
        else:
            raise ValueError(mode)

    def child_row(self, depth: int, tok: int, parent_tok: Optional[int] = None) -> Optional[int]:
        if depth >= self.gamma:          # reading R7
            return None
        if self.mode == "marginal":      # DDTree: every node shares q_{t+depth+1}
            return depth
        try:
            m = self.top_m[depth - 1].index(tok)   # is v = x^(m)_{t+depth} ?
        except ValueError:
            return None                  # leaf: outside the M-ary tree
        if self.mode == "marginal_mary":
            return depth
        if not self.two_prev:
            return 1 + (depth - 1) * self.M + m    # row of q'^(m)_{t+depth+1}
        if depth == 1:                             # reading R13: (x^(m)_{t+1}, x_t)
            return 1 + m
        mp = self.top_m[depth - 2].index(parent_tok)   # the parent was expanded: in the M-ary tree
        return 1 + self.M + (depth - 2) * self.M * self.M + m * self.M + mp


def build_tree_literal(src: ChildSource, root_tok: int, B: int, keep: Optional[int] = None) -> Tree:
    """Algorithm 1 Part 2 as written: every expansion pushes the whole distribution (or its
    top `keep` entries, reading R5) into the queue; B pops. Small vocabularies only."""
    heap = []

    def push_row(row_idx: int, parent: int, parent_score: float, depth: int):
        lp = src.rows[row_idx]
        cand = ranked(lp) if keep is None else ranked(lp, keep)
        for v in cand:
            s = parent_score + lp[v]
            heapq.heappush(heap, (-s, depth, parent, int(v), row_idx))

    toks, parents, depths, scores, rows = [root_tok], [-1], [0], [0.0], [-1]
    push_row(src.root_row, 0, 0.0, 1)
    pops = []
    while len(toks) < B + 1 and heap:
        negs, dep, par, v, r = heapq.heappop(heap)
        node = len(toks)
        toks.append(v); parents.append(par); depths.append(dep); scores.append(-negs); rows.append(r)
        pops.append((-negs, dep, par, v))
        cr = src.child_row(dep, v, toks[par])
        if cr is not None:
            push_row(cr, node, -negs, dep + 1)
    return _finish(toks, parents, depths, scores, rows, B, pops)


def build_tree_lazy(src: ChildSource, root_tok: int, B: int, keep: Optional[int] = None) -> Tree:
    """The same selection with a lazy queue: a distribution enters the queue as its best
    remaining entry, and popping rank k of a row pushes rank k+1 of the same row for the same
    parent. Equivalent to build_tree_literal because rank k+1 never precedes rank k in the
    queue order of reading R8 (equal score, same depth and parent, larger token id, or a
    lower score). Needed for full vocabularies."""
    order_cache = {}

    def order(row_idx):
        if row_idx not in order_cache:
            o = ranked(src.rows[row_idx])
            order_cache[row_idx] = o if keep is None else o[:keep]
        return order_cache[row_idx]

    heap = []

    def push(row_idx, parent, parent_score, depth, rank):
        o = order(row_idx)
        if rank < len(o):
            v = int(o[rank])
            s = parent_score + src.rows[row_idx][v]
            heapq.heappush(heap, (-s, depth, parent, v, row_idx, rank, parent_score))

    toks, parents, depths, scores, rows = [root_tok], [-1], [0], [0.0], [-1]
    push(src.root_row, 0, 0.0, 1, 0)
    pops = []
    while len(toks) < B + 1 and heap:
        negs, dep, par, v, r, rank, pscore = heapq.heappop(heap)
        node = len(toks)
        toks.append(v); parents.append(par); depths.append(dep); scores.append(-negs); rows.append(r)
        pops.append((-negs, dep, par, v))
        push(r, par, pscore, dep, rank + 1)          # next sibling in the same row
        cr = src.child_row(dep, v, toks[par])
        if cr is not None:
            push(cr, node, -negs, dep + 1, 0)        # best child of the new node
    return _finish(toks, parents, depths, scores, rows, B, pops)


def _finish(toks, parents, depths, scores, rows, B, pops) -> Tree:
    n = len(toks)
    pad = B + 1 - n
    t = Tree(tok=np.array(toks + [-1] * pad, dtype=np.int64),
             parent=np.array(parents + [-1] * pad, dtype=np.int64),
             depth=np.array(depths + [-1] * pad, dtype=np.int64),
             score=np.array(scores + [NEG_INF] * pad, dtype=np.float64),
             row=np.array(rows + [-1] * pad, dtype=np.int64),
             underfull=pad > 0, pops=pops)
    return t


# ---------------------------------------------------------------------------------------
# tree-attention mask and position ids
# ---------------------------------------------------------------------------------------


def tree_mask(parent: np.ndarray, depth: np.ndarray, root_pos: int):
    """mask[i, j] = 1 iff node j is node i or one of its ancestors (node i may attend to
    j in the verifier's single pass over the tree); pos[i] = root_pos + depth[i]. Missing
    nodes (parent == -1 beyond the root) get an all-zero row and column and pos -1."""
    n = parent.shape[0]
    present = np.zeros(n, dtype=bool)
    present[0] = True
    present[1:] = parent[1:] >= 0
    mask = np.zeros((n, n), dtype=np.uint8)
    for i in range(n):
        if not present[i]:
            continue
        j = i
        while j >= 0:
            mask[i, j] = 1
            j = parent[j] if j > 0 else -1
    pos = np.where(present, root_pos + depth, -1).astype(np.int64)
    return mask, pos

def accept_walk(tok: np.ndarray, parent: np.ndarray, verifier_tok: np.ndarray):
    """Verification of a drafted tree by an equality check, and the step's block efficiency.

    Sec. 3: token selection is deterministic, so a drafted token is accepted exactly when it
    equals the verifier's own next token at that position. verifier_tok[i] is the verifier's
    next token at the position of node i (its choice after the path root..i). Starting at the
    root, the walk moves to the child of the current node whose token equals the verifier's
    token there, while such a child exists (children of one node carry distinct tokens; if an
    invalid tree repeats one, the smallest node index is taken). Sec. 4: block efficiency tau
    counts the accepted tokens plus the verifier's residual token.

    Returns (path, bonus): path = accepted node indices, root first (the tree rows whose KV
    entries the verifier keeps); bonus = verifier_tok at the last accepted node. The step
    accepts len(path) - 1 drafted tokens and gains tau = len(path) tokens. Missing nodes
    (parent -1 beyond the root) are never children.
    """
    n = len(tok)
    children = [[] for _ in range(n)]
    for c in range(1, n):
        if parent[c] >= 0:
            children[int(parent[c])].append(c)
    path = [0]
    cur = 0
    while True:
        match = [c for c in children[cur] if tok[c] == verifier_tok[cur]]
        if not match:
            break
        cur = match[0]
        path.append(cur)
    return path, int(verifier_tok[cur])


# ---------------------------------------------------------------------------------------
# the whole drafting step
# ---------------------------------------------------------------------------------------


@dataclass
class SeqResult:
    s1_logp: np.ndarray      # [gamma, V]
    top_ids: np.ndarray      # [gamma, K1]
    top_logp: np.ndarray     # [gamma, K1]
    h_prime: Optional[np.ndarray]   # [R, d]
    s2_logp: Optional[np.ndarray]   # [R, V]
    child_ids: Optional[np.ndarray]   # [R, K2]
    child_logp: Optional[np.ndarray]  # [R, K2]
    tree: Tree
    mask: np.ndarray
    pos: np.ndarray
    approx: str = "swiglu"


def draft_sequence(H: np.ndarray, root_tok: int, root_pos: int, W: dict, *, M: int, K2: int,
                   B: int, temperature: float = 1.0, eps: float = 1e-6, mode: str = "ar",
                   emulate_bf16: bool = False, keep: Optional[int] = None,
                   literal: bool = False, approx: str = "swiglu",
                   root_prev: Optional[int] = None) -> SeqResult:
    """One sequence through Algorithm 1 (both parts) and the mask. W holds float64 arrays
    lm_head [V,d], embed [V,d], norm_h [d], norm_e [d], w_gate [I,2d], w_up [I,2d],
    w_down [d,I] (approx "swiglu"; [I,3d] gate/up for "swiglu_2prev", reading R13, which also
    needs root_prev, the token before the root) or w_lin [d,2d] (approx "linear", reading
    R12). `keep` truncates every child list (reading R5); None = whole distributions."""
    gamma = H.shape[0]
    K1 = max(M, K2)
    s1_logp, top_ids, top_logp = stage1(H, W["lm_head"], temperature, K1)
    hp = s2 = cids = clp = None
    if mode == "ar":
        hp, s2 = stage2(H, root_tok, top_ids, W, M, temperature, eps, emulate_bf16, approx, root_prev)
        cids = np.stack([ranked(r, K2) for r in s2])
        clp = np.take_along_axis(s2, cids, axis=1)
    src = ChildSource(mode, gamma, M, top_ids, s1_logp, s2, approx)
    builder = build_tree_literal if literal else build_tree_lazy
    tree = builder(src, int(root_tok), B, keep)
    mask, pos = tree_mask(tree.parent, tree.depth, int(root_pos))
    return SeqResult(s1_logp, top_ids, top_logp, hp, s2, cids, clp, tree, mask, pos, approx)


def weights_f64(inputs: dict, to_f64) -> dict:
    keys = ("lm_head", "embed", "norm_h", "norm_e", "w_gate", "w_up", "w_down", "w_lin")
    return {k: to_f64(inputs[k]) for k in keys if inputs.get(k) is not None}


# ---------------------------------------------------------------------------------------
# selection margins (used by parity tests to decide where structure must match exactly)
# ---------------------------------------------------------------------------------------


def topk_margin(values: np.ndarray, k: int) -> float:
    """Gap between the k-th and (k+1)-th largest entries (inf if there is no k+1-th)."""
    if k >= values.shape[-1]:
        return np.inf
    part = -np.partition(-values, k)[: k + 1]
    part = np.sort(part)[::-1]
    return float(part[k - 1] - part[k])


def selection_margins(res: SeqResult, M: int, K2: int, B: int, mode: str = "ar"):
    """(set_margin, order_margin): the smallest gaps that decide the tree.

    set_margin decides WHICH nodes are selected: the per-depth gap at the M-th stage-1
    candidate for depths 1..gamma-1 (it fixes the M-ary tree and the stage-2 conditioning;
    unused by DDTree), the gap between the B-th pop and the best candidate left out, and
    the gap at the K2-th entry of every child list when K2 < B truncates.
    order_margin additionally covers the gaps between consecutive pops, which fix the node
    numbering (pop order) and hence the parent indices."""
    gamma = res.top_ids.shape[0]
    gaps = []
    if mode != "marginal":
        gaps += [topk_margin(r, M) for r in res.s1_logp[: gamma - 1]]
    if K2 < B:
        rows = res.s2_logp if mode == "ar" else res.s1_logp
        gaps += [topk_margin(r, K2) for r in rows]
    scores = [p[0] for p in res.tree.pops]
    nxt = _next_score_after(res, M, K2, B, mode)
    if nxt is not None and scores:
        gaps.append(scores[-1] - nxt)
    set_margin = float(min(gaps)) if gaps else np.inf
    adj = [a - b for a, b in zip(scores, scores[1:])]
    order_margin = float(min([set_margin] + adj))
    return set_margin, order_margin


def _next_score_after(res: SeqResult, M, K2, B, mode):
    """Score of the (B+1)-th pop (the best candidate left out), or None."""
    src = ChildSource(mode, res.top_ids.shape[0], M, res.top_ids, res.s1_logp, res.s2_logp, res.approx)
    t = build_tree_lazy(src, int(res.tree.tok[0]), B + 1, keep=K2 if K2 < B else None)
    if len(t.pops) <= B:
        return None
    return t.pops[B][0]


# ---------------------------------------------------------------------------------------
# brute force (tiny vocabularies): the eligible universe and exhaustive prefix-closed sets
# ---------------------------------------------------------------------------------------


def eligible_universe(src: ChildSource, max_nodes: int = 200000):
    """Every node Algorithm 1 could ever emit: (score, depth, parent_path, tok, path) with
    path the token tuple from depth 1. Children exist only below expandable nodes."""
    out = []
    frontier = [((), 0.0, src.root_row, 1)]
    while frontier:
        path, pscore, row, depth = frontier.pop()
        lp = src.rows[row]
        for v in range(lp.shape[0]):
            s = pscore + lp[v]
            p = path + (v,)
            out.append((s, depth, p))
            if len(out) > max_nodes:
                raise RuntimeError("universe too large")
            cr = src.child_row(depth, v, path[-1] if path else None)
            if cr is not None:
                frontier.append((p, s, cr, depth + 1))
    return out


def tree_paths(t: Tree) -> List[tuple]:
    """Token path (from depth 1) of every non-root node."""
    paths = [()]
    for i in range(1, t.tok.shape[0]):
        if t.parent[i] < 0:
            continue
        paths.append(paths[t.parent[i]] + (int(t.tok[i]),))
    return paths[1:]


def best_prefix_closed_value(universe, B: int) -> float:
    """Maximum over all prefix-closed node sets of size B of the summed path probability
    (the OPT-Tree objective of Sec. 3: the expected number of accepted tokens), by
    exhaustive recursive enumeration. Tiny universes only."""
    prob = {p: float(np.exp(s)) for s, _, p in universe}
    children = {}
    for _, _, p in universe:
        children.setdefault(p[:-1], []).append(p)
    best = [0.0]

    def rec(chosen_val, available, k):
        if k == 0:
            best[0] = max(best[0], chosen_val)
            return
        # pick the next node among available ones in canonical order to avoid repeats
        for idx, node in enumerate(available):
            rest = available[idx + 1:] + children.get(node, [])
            rec(chosen_val + prob[node], rest, k - 1)

    rec(0.0, list(children.get((), [])), B)
    return best[0]
