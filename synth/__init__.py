"""Seeded synthetic workloads for the TreeFlash drafting path.

This module only draws inputs. It holds none of the method's arithmetic (no LM head, no
approximator, no softmax over a model's logits, no tree search), so that the fp64 oracle
and the CUDA path can both be fed from it without sharing any code with each other.

What the inputs stand in for: the paper measures drafting on DFlash/TreeFlash checkpoints
with Qwen3 verifiers over MATH-500, GSM8K, HumanEval, MBPP and MT-Bench (Sec. 4,
"Datasets" and "Inference Parameters"). None of those models or datasets are used here.
Instead every tensor is i.i.d. Gaussian with the paper's shapes (block size gamma, M
candidates per depth, budget B, temperature T = 1, bf16) and the Qwen3 vocabulary size;
the drafter hidden states are scaled so that the marginal next-token distributions have a
chosen entropy (by default a ramp from 2 nats at depth 1 to 4 nats at depth gamma, the
depth-growing uncertainty of Fig. 3 / Fig. 4).

Entropy calibration: for W_lm with i.i.d. N(0, w_std^2) entries and a fixed hidden
vector h, the logits W_lm h are i.i.d. N(0, w_std^2 |h|^2) across the vocabulary. So the
generator picks the logit scale sigma whose Gaussian-logit softmax has the target entropy
(bisection over a fixed seeded N(0,1) sample of size V) and draws h = s * N(0, 1) with
s = sigma / (w_std * sqrt(d)). This is a statement about Gaussian samples, not a call of
the method.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional, Tuple

import numpy as np
import torch

__all__ = ["Config", "CONFIGS", "get_config", "make_inputs", "gaussian_logit_scale"]


@dataclasses.dataclass(frozen=True)
class Config:
    name: str
    batch: int
    d: int
    V: int
    I: int
    gamma: int
    M: int
    K2: int
    B: int
    dtype: str = "bf16"            # "bf16" or "f32": storage and input type of every tensor
    mode: str = "ar"               # "ar" (TreeFlash), "marginal" (DDTree), "marginal_mary"
    approx: str = "swiglu"         # stage-2 approximator: "swiglu" (Eq. 1), or the ablations'
                                   # "linear" and "swiglu_2prev" (two previous tokens)
    temperature: float = 1.0
    rms_eps: float = 1e-6
    seed: int = 0
    w_std: float = 0.02            # W_lm, E, W_gate, W_up
    wd_std: float = 0.02           # W_down, and W_lin of the linear approximator
    h_std: float = 1.0             # used when h_entropy is None: h ~ N(0, h_std^2)
    h_entropy: Optional[Tuple[float, float]] = None  # (nats at depth 1, nats at depth gamma)

    @property
    def R(self) -> int:
        """Stage-2 rows per sequence: one for depth 1, M for each depth 2..gamma (with two
        previous tokens: M for depth 2 and M^2 for each depth 3..gamma)."""
        if self.approx == "swiglu_2prev" and self.mode == "ar":
            return 1 if self.gamma == 1 else 1 + self.M + self.M * self.M * (self.gamma - 2)
        return 1 + self.M * (self.gamma - 1)

    @property
    def K1(self) -> int:
        return max(self.M, self.K2)

    def replace(self, **kw) -> "Config":
        return dataclasses.replace(self, **kw)


_Q8 = dict(d=4096, V=151936, I=4096, gamma=16, dtype="bf16", h_entropy=(2.0, 4.0))

CONFIGS = {
    # batch 1, d=128, V=2048, MLP 2d->512->d, gamma=4, top-4 per depth, B=12, all N(0, 0.02)
    "tiny_f32": Config("tiny_f32", batch=1, d=128, V=2048, I=512, gamma=4, M=4, K2=12, B=12,
                       dtype="f32", h_std=0.02),
    # the same at V=16, small enough for brute-force enumeration
    "tiny_v16": Config("tiny_v16", batch=1, d=128, V=16, I=512, gamma=4, M=4, K2=12, B=12,
                       dtype="f32", h_std=0.02),
    # tiny with peaked marginals (so that the tree grows in depth) and a strong approximator
    "tiny_peaked": Config("tiny_peaked", batch=1, d=128, V=2048, I=512, gamma=4, M=4, K2=12,
                          B=12, dtype="f32", h_entropy=(1.0, 2.0), wd_std=0.5),
    # Qwen3-8B shape, gamma=16, M=8, B=32
    "q8_b32": Config("q8_b32", batch=1, M=8, K2=32, B=32, **_Q8),
    # Qwen3-8B shape, gamma=16, M=16, B=64 (the measured workload)
    "q8_b64": Config("q8_b64", batch=1, M=16, K2=64, B=64, **_Q8),
    # 32 independent sequences of the q8_b32 shape in one launch
    "batch32": Config("batch32", batch=32, M=8, K2=32, B=32, **_Q8),
    # wide model, batch 8, peaked (~1 nat) and flat (~5 nat) hidden-state regimes
    "wide_peaked": Config("wide_peaked", batch=8, d=5120, V=151936, I=5120, gamma=16, M=16,
                          K2=64, B=64, h_entropy=(1.0, 1.0)),
    "wide_flat": Config("wide_flat", batch=8, d=5120, V=151936, I=5120, gamma=16, M=16,
                        K2=64, B=64, h_entropy=(5.0, 5.0)),
    # large draft budget (Fig. 5) with exact per-row lists (K2 = B), and wide branching (Fig. 6)
    "q8_b512": Config("q8_b512", batch=1, M=16, K2=512, B=512, **_Q8),
    "q8_m64": Config("q8_m64", batch=1, M=64, K2=64, B=64, **_Q8),
    # the q8_b64 step with the "w/ Linear" ablation's approximator (Sec. 4, Table 3)
    "q8_b64_linear": Config("q8_b64_linear", batch=1, M=16, K2=64, B=64, approx="linear", **_Q8),
    # the q8_b32 and q8_b64 steps with the two-previous-token approximator (the "w/ 2-prev"
    # ablation): 1 + M + M^2 (gamma - 2) = 905 / 3601 stage-2 rows
    "q8_b32_2prev": Config("q8_b32_2prev", batch=1, M=8, K2=32, B=32, approx="swiglu_2prev", **_Q8),
    "q8_b64_2prev": Config("q8_b64_2prev", batch=1, M=16, K2=64, B=64, approx="swiglu_2prev", **_Q8),
    # the q8_b64 step with the approximator width the paper's parameter counts imply for a
    # Qwen3-8B verifier (its intermediate size, I = 12288)
    "q8_b64_paper_i": Config("q8_b64_paper_i", batch=1, M=16, K2=64, B=64, **dict(_Q8, I=12288)),
    # the q8_b64 step with the vocabulary cut to 32768 (W_lm 268 MB, still twice the L2):
    # small enough for multi-pass profiler captures
    "prof_v32k": Config("prof_v32k", batch=1, M=16, K2=64, B=64, **dict(_Q8, V=32768)),
}


def get_config(name: str, **overrides) -> Config:
    cfg = CONFIGS[name]
    return cfg.replace(**overrides) if overrides else cfg


def _softmax_entropy_of_scaled(sample: np.ndarray, sigma: float) -> float:
    # entropy (nats) of softmax(sigma * g) for a fixed Gaussian sample g
    z = sigma * sample
    z = z - z.max()
    p = np.exp(z)
    s = p.sum()
    p /= s
    nz = p > 0
    return float(-(p[nz] * np.log(p[nz])).sum())


def gaussian_logit_scale(V: int, target_nats: float, seed: int = 12345) -> float:
    """Logit standard deviation sigma such that V i.i.d. N(0, sigma^2) logits have a softmax
    entropy of `target_nats` (bisection on a fixed seeded sample)."""
    if not (0.0 < target_nats < math.log(V)):
        raise ValueError("target entropy must lie in (0, log V)")
    g = np.random.default_rng(seed).standard_normal(V)
    lo, hi = 0.0, 1.0
    while _softmax_entropy_of_scaled(g, hi) > target_nats:
        hi *= 2.0
        if hi > 1e6:
            raise RuntimeError("entropy calibration did not bracket")
    for _ in range(60):
        mid = 0.5 * (lo + hi)
        if _softmax_entropy_of_scaled(g, mid) > target_nats:
            lo = mid
        else:
            hi = mid
    return 0.5 * (lo + hi)


def hidden_scales(cfg: Config) -> np.ndarray:
    """Per-depth standard deviation of the drafter hidden states."""
    if cfg.h_entropy is None:
        return np.full(cfg.gamma, cfg.h_std)
    h0, h1 = cfg.h_entropy
    out = np.empty(cfg.gamma)
    for i in range(cfg.gamma):
        t = 0.0 if cfg.gamma == 1 else i / (cfg.gamma - 1)
        sigma = gaussian_logit_scale(cfg.V, h0 + (h1 - h0) * t)
        out[i] = sigma / (cfg.w_std * math.sqrt(cfg.d))
    return out


def _randn(gen: torch.Generator, shape, std: float, dtype: torch.dtype) -> torch.Tensor:
    t = torch.randn(*shape, generator=gen, dtype=torch.float32)
    t.mul_(std)
    return t.to(dtype)


def make_inputs(cfg: Config, seed: Optional[int] = None) -> dict:
    """All inputs of one drafting step as CPU tensors of the config's dtype.

    Keys: hidden [b, gamma, d], lm_head [V, d], embed [V, d], norm_h [d], norm_e [d],
    w_gate [I, 2d], w_up [I, 2d], w_down [d, I], root_tok [b] int32, root_pos [b] int32,
    h_scale [gamma] float64 (the per-depth hidden-state std that was used), and for the linear
    approximator w_lin [d, 2d] ~ N(0, wd_std^2), drawn last so that every other tensor is the
    same as for the SwiGLU configuration of the same shape and seed. For the two-previous-token
    approximator w_gate and w_up are [I, 3d]: the SwiGLU configuration's [I, 2d] matrices with
    d more columns (for the second previous token) drawn last, and root_prev [b] int32 is the
    token before each root.
    """
    seed = cfg.seed if seed is None else seed
    dt = torch.float32 if cfg.dtype == "f32" else torch.bfloat16
    g = torch.Generator().manual_seed(seed)
    d, V, I = cfg.d, cfg.V, cfg.I
    lm_head = _randn(g, (V, d), cfg.w_std, dt)
    embed = _randn(g, (V, d), cfg.w_std, dt)
    w_gate = _randn(g, (I, 2 * d), cfg.w_std, dt)
    w_up = _randn(g, (I, 2 * d), cfg.w_std, dt)
    w_down = _randn(g, (d, I), cfg.wd_std, dt)
    scales = hidden_scales(cfg)
    base = torch.randn(cfg.batch, cfg.gamma, d, generator=g, dtype=torch.float32)
    base.mul_(torch.tensor(scales, dtype=torch.float32).view(1, cfg.gamma, 1))
    hidden = base.to(dt)
    root_tok = torch.randint(0, V, (cfg.batch,), generator=g, dtype=torch.int64).to(torch.int32)
    root_pos = (torch.arange(cfg.batch, dtype=torch.int32) * 7 + 1000).to(torch.int32)
    out = dict(hidden=hidden, lm_head=lm_head, embed=embed,
               norm_h=torch.ones(d, dtype=dt), norm_e=torch.ones(d, dtype=dt),
               w_gate=w_gate, w_up=w_up, w_down=w_down,
               root_tok=root_tok, root_pos=root_pos, h_scale=scales)
    if cfg.approx == "linear":
        out["w_lin"] = _randn(g, (d, 2 * d), cfg.wd_std, dt)
    elif cfg.approx == "swiglu_2prev" and cfg.mode == "ar":
        out["w_gate"] = torch.cat([w_gate, _randn(g, (I, d), cfg.w_std, dt)], dim=1).contiguous()
        out["w_up"] = torch.cat([w_up, _randn(g, (I, d), cfg.w_std, dt)], dim=1).contiguous()
        out["root_prev"] = torch.randint(0, V, (cfg.batch,), generator=g, dtype=torch.int64).to(torch.int32)
    return out


def to_f64(t: torch.Tensor) -> np.ndarray:
    """Exact widening of a float tensor (bf16 or f32) to a float64 numpy array."""
    return t.detach().to(torch.float64).cpu().numpy()
