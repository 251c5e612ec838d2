"""Benchmark of the TreeFlash drafting hot path: one step = one whole draft-tree build.

A step runs every call of the path on the batch of the measured workload (Qwen3-8B shape,
gamma=16, M=16, B=64, batch 1): the stage-1 LM-head pass and its top-k merge, the
AR-approximator (Eq. 1), the stage-2 LM-head pass and merge, the best-first tree build and the
mask. Inputs are seeded synthetic tensors already resident in HBM; W_lm (1.245 GB) is streamed
twice per step, far beyond the 129 MB L2, so nothing is flushed between steps.

Output: one JSON line on rank 0 (see --help for the arms). `value` is timed over K whole steps
with no instrumentation between them. The `roofline` object covers the dominant kernel (the
fused LM-head pass): algorithmic bytes per launch (|W_lm| + the activation rows) over its average
CUDA-event duration, from a second pass of the same steps with events around the two LM-head
launches. `gpu_launches` is the library's own count of kernels launched in the timed region. `e2e` is the same metric
through tf_draft_tree_host with the step's inputs and outputs in pinned host memory, copies
inside the timed region, on a created stream (the library then replays the step as a CUDA graph
captured at the first call). `cpu_baseline` is the fp64 oracle on the host cores on a bounded sample.
`torch_eager` times the same step written with PyTorch library calls (logits materialised,
Part 2 as a host loop, as in the paper's implementation): a reference point, not a competitor.

Multi-GPU (torchrun, one rank per GPU): every rank builds its own trees (independent replicas,
no collective on the data path); value = all trees built / max over ranks of the timed span.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "µs per draft-tree build (trees/s) at Qwen3-8B shape, B=32/64; % of HBM roofline"
WORKLOAD = "q8_b64"
FALLBACK_HBM_GBS = 6800.0
NOMINAL_HBM_GBS = 8000.0          # GB300 HBM3e, nominal (~8 TB/s); the measured copy rate is the peak
FALLBACK_BF16_TFLOPS_SUSTAINED = 1700.0


# ------------------------------------------------------------------------------ distributed

def dist_env():
    return int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")), \
        int(os.environ.get("LOCAL_RANK", "0"))


def init_dist(backend: str):
    import torch.distributed as dist
    rank, world, _ = dist_env()
    if world > 1 and not dist.is_initialized():
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        dist.init_process_group(backend=backend, rank=rank, world_size=world)
    return rank, world


def barrier(world: int, device=None):
    if world > 1:
        import torch.distributed as dist
        if device is not None and dist.get_backend() == "nccl":
            dist.barrier(device_ids=[device.index])
        else:
            dist.barrier()


def max_over_ranks(x: float, world: int, device=None) -> float:
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device if dist.get_backend() == "nccl" else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ------------------------------------------------------------------------------ clocks

class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons while the timed region runs."""

    FIELDS = "clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown," \
             "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown," \
             "clocks_event_reasons.sw_power_cap"

    def __init__(self, index: int):
        self.index = index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        time.sleep(0.25)
        return self

    def __exit__(self, *exc):
        self.out = ""
        if self.proc is not None:
            time.sleep(0.15)
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                self.out, _ = self.proc.communicate()

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in (self.out or "").splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 7:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for n, v in zip(names, parts[3:7]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        # samples under load: the upper part of the trace (the sampler brackets the region)
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# ------------------------------------------------------------------------------ helpers

def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        d = json.load(open(p))
        return float(d["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return FALLBACK_HBM_GBS, "fallback"


def tensor_peak():
    """bf16 dense tensor rate for a kernel timed inside a long step (the sustained figure)."""
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        return float(json.load(open(p))["bf16_tflops_sustained"]), "measured"
    except (OSError, KeyError, ValueError):
        return FALLBACK_BF16_TFLOPS_SUSTAINED, "fallback"


def kernel_source_hash():
    h = hashlib.sha256()
    for f in ("tc_gemm.cu", "tc_ptx.cuh", "common.cuh"):
        h.update(open(os.path.join(ROOT, "paper_2606_03819_gb300", "csrc", f), "rb").read())
    return h.hexdigest()[:16]


def profiled_traffic(workload: str):
    """dram bytes per launch of the LM-head pass from the committed ncu summary, or None when
    the kernel sources changed since the counters were taken or the summary covers another
    workload (it was scaled to the measured one)."""
    p = os.path.join(ROOT, "profiles", "lmhead_traffic.json")
    try:
        d = json.load(open(p))
    except (OSError, ValueError):
        return None
    if d.get("source_hash") != kernel_source_hash() or not str(d.get("scaled_to", "")).startswith(workload + " "):
        return None
    return d.get("dram_bytes_per_launch")


def algorithmic_bytes(cfg):
    """Bytes a tree build must move at least: W_lm twice (stage 2 needs the global stage-1
    top-M first, and W_lm is ~10x the L2), the approximator's matrices (the linear variant's
    W_lin alone), the gathered embedding rows and the hidden states. Outputs are ignored."""
    e = 2 if cfg.dtype == "bf16" else 4
    lm = cfg.V * cfg.d * e
    if cfg.approx == "linear":
        mlp = cfg.d * 2 * cfg.d * e                    # W_lin [d, 2d]
    else:
        k_in = (3 if cfg.approx == "swiglu_2prev" else 2) * cfg.d
        mlp = (2 * cfg.I * k_in + cfg.d * cfg.I) * e   # W_gate, W_up [I, 2d or 3d]; W_down [d, I]
    rows = cfg.batch * cfg.R
    gathered = rows * cfg.d * e
    hidden = cfg.batch * cfg.gamma * cfg.d * e
    return 2 * lm + mlp + gathered + hidden, lm


def lmhead_roofline(cfg, n1, n2, lm1_ms, lm2_ms, hbm_peak, tc_peak, traffic, timing):
    """The `roofline` object of the dominant kernel, the LM-head pass (one launch over the n1
    stage-1 rows, one over the n2 stage-2 rows; lm1_ms / lm2_ms their mean CUDA-event times).
    Per launch it moves |W_lm| + rows * d * 2 bytes and does 2 * rows * V * d flops. The pass
    is bound by HBM unless the bf16 contraction at the sustained tensor rate takes longer than
    streaming those bytes at the copy rate (many stage-2 rows: batched sequences, two previous
    tokens); then it is reported against the tensor rate, with the HBM figures beside it.
    hbm_peak, tc_peak: (value, kind) in GB/s and TFLOP/s."""
    (peak, peak_kind), (tc, tc_kind) = hbm_peak, tc_peak
    _, lm_bytes = algorithmic_bytes(cfg)
    nbytes = [lm_bytes + n1 * cfg.d * 2, lm_bytes + n2 * cfg.d * 2]
    flops = [2.0 * n1 * cfg.V * cfg.d, 2.0 * n2 * cfg.V * cfg.d]
    avg_s = (lm1_ms + lm2_ms) / 2 / 1e3
    gbs = sum(nbytes) / 2 / avg_s / 1e9
    hbm = {"bound": "hbm", "kernel": "tc_gemm_kernel<LMHEAD> (stage-1 and stage-2 launches)",
           "achieved": gbs, "peak": peak, "unit": "GB/s", "frac": gbs / peak, "traffic": traffic,
           "frac_nominal": gbs / NOMINAL_HBM_GBS,
           "peak_kind": peak_kind, "launch_ms": {"stage1": lm1_ms, "stage2": lm2_ms},
           "bytes_per_launch": {"stage1": nbytes[0], "stage2": nbytes[1]},
           "flops_per_launch": {"stage1": flops[0], "stage2": flops[1]}, "timing": timing}
    if sum(flops) / (tc * 1e12) <= sum(nbytes) / (peak * 1e9):
        return hbm
    tflops = sum(flops) / 2 / avg_s / 1e12
    out = dict(hbm, bound="tensor", achieved=tflops, peak=tc, unit="TFLOP/s", frac=tflops / tc,
               peak_kind=f"{tc_kind} bf16 sustained")
    out["hbm"] = {"achieved": gbs, "peak": peak, "unit": "GB/s", "frac": gbs / peak}
    return out


# ------------------------------------------------------------------------------ library-call reference

def torch_eager_tree(cfg, w, hidden, root_tok):
    """The drafting step written with PyTorch library calls, as a timing reference point (the
    way the paper's own implementation runs Part 1, with Part 2 as a host loop; App. B):
    matmuls in the tensors' dtype, log_softmax and topk on full fp32 logits (which reach
    memory), Eq. 1 as torch ops, then the best-first selection with heapq on the host.
    TreeFlash mode with the SwiGLU approximator only. Returns per sequence (tok, parent, depth,
    score) lists of the B + 1 nodes in pop order. Not used by the library; runs on any device."""
    import heapq

    import torch
    import torch.nn.functional as F
    b, g, M, K2, B, d = cfg.batch, cfg.gamma, cfg.M, cfg.K2, cfg.B, cfg.d
    K1 = max(M, K2)
    W = w["lm_head"]
    logp1 = torch.log_softmax((hidden.reshape(b * g, d) @ W.T).float() / cfg.temperature, dim=-1)
    _, i1 = torch.topk(logp1, K1, dim=-1)
    i1 = i1.view(b, g, K1)
    # stage-2 rows: depth 1 on the root token, depth i on each candidate of depth i - 1
    depth_of_row = torch.tensor([0] + [i for i in range(1, g) for _ in range(M)], device=hidden.device)
    prev = torch.cat([root_tok.view(b, 1).long(), i1[:, : g - 1, :M].reshape(b, (g - 1) * M)], dim=1)
    h_rows = hidden[:, depth_of_row, :]

    def rms(x, wt):
        xf = x.float()
        return (xf * torch.rsqrt(xf.pow(2).mean(-1, keepdim=True) + cfg.rms_eps) * wt.float()).to(x.dtype)
    x = torch.cat([rms(h_rows, w["norm_h"]), rms(w["embed"][prev], w["norm_e"])], dim=-1)
    a = (F.silu((x @ w["w_gate"].T).float()) * (x @ w["w_up"].T).float()).to(x.dtype)
    hp = (h_rows.float() + (a @ w["w_down"].T).float()).to(x.dtype)
    logp2 = torch.log_softmax((hp.reshape(b * cfg.R, d) @ W.T).float() / cfg.temperature, dim=-1)
    v2, i2 = torch.topk(logp2, K2, dim=-1)
    top_m = i1[:, :, :M].cpu().tolist()
    v2 = v2.view(b, cfg.R, K2).cpu().tolist()
    i2 = i2.view(b, cfg.R, K2).cpu().tolist()
    trees = []
    for s in range(b):
        toks, pars, deps, scores = [int(root_tok[s])], [-1], [0], [0.0]
        heap = [(-v2[s][0][0], 1, 0, 0, 0, 0.0)]   # (-score, depth, parent, row, rank, parent score)
        while heap and len(toks) < B + 1:
            negs, dep, par, row, rank, psc = heapq.heappop(heap)
            node = len(toks)
            tok = i2[s][row][rank]
            toks.append(tok)
            pars.append(par)
            deps.append(dep)
            scores.append(-negs)
            if rank + 1 < K2:
                heapq.heappush(heap, (-(psc + v2[s][row][rank + 1]), dep, par, row, rank + 1, psc))
            if dep < g and tok in top_m[s][dep - 1]:
                crow = 1 + (dep - 1) * M + top_m[s][dep - 1].index(tok)
                heapq.heappush(heap, (-(-negs + v2[s][crow][0]), dep + 1, node, crow, 0, -negs))
        trees.append((toks, pars, deps, scores))
    return trees


def time_torch_eager(cfg, w, hidden, root_tok, steps: int):
    """Wall-clock trees/s of torch_eager_tree on the GPU (each step ends with the host loop,
    so it synchronises)."""
    import torch
    for _ in range(2):
        torch_eager_tree(cfg, w, hidden, root_tok)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(steps):
        torch_eager_tree(cfg, w, hidden, root_tok)
    torch.cuda.synchronize()
    t = (time.perf_counter() - t0) / steps
    return {"value": cfg.batch / t, "unit": "trees/s", "ms_per_step": t * 1e3, "steps": steps,
            "what": "torch library calls on the GPU (bf16 matmuls, fp32 logits in HBM, log_softmax, topk) "
                    "plus a heapq best-first loop on the host; a reference point, not the product path"}


# ------------------------------------------------------------------------------ oracle timing

class OracleSample:
    """The fp64 oracle on one sequence of the workload, with the vocabulary cut to a fraction
    (the LM-head passes, log-softmax and sorting scale with V; the approximator does not).
    Weights are widened to float64 once, outside any timing."""

    def __init__(self, cfg, inp):
        import synth
        self.cfg = cfg
        keys = ("embed", "norm_h", "norm_e") + (("w_lin",) if cfg.approx == "linear" else ("w_gate", "w_up", "w_down"))
        self.W = {k: synth.to_f64(inp[k]) for k in keys}
        self.lm = synth.to_f64(inp["lm_head"])
        self.H = synth.to_f64(inp["hidden"][0])
        self.root = int(inp["root_tok"][0])
        self.root_prev = int(inp["root_prev"][0]) if inp.get("root_prev") is not None else None

    def run(self, fraction: float):
        """Returns (seconds for the sample, estimated seconds for a whole tree, vocabulary used)."""
        import numpy as np
        from oracle import treeflash_oracle as O
        cfg = self.cfg
        Vs = max(cfg.K2 + cfg.M, int(math.ceil(cfg.V * fraction)))
        W = dict(self.W, lm_head=self.lm[:Vs])
        root = self.root % Vs
        rprev = None if self.root_prev is None else self.root_prev % Vs
        no_top = np.zeros((cfg.gamma, cfg.M), dtype=np.int64)
        hid, prev = O.stage2_conditioning(cfg.gamma, cfg.M, root, no_top)
        t0 = time.perf_counter()
        if cfg.approx == "swiglu_2prev":
            hid, prev, prev2 = O.stage2_conditioning_2prev(cfg.gamma, cfg.M, root, rprev, no_top)
            O.ar_approximator(self.H[hid], W["embed"][prev], W["norm_h"], W["norm_e"], W["w_gate"], W["w_up"],
                              W["w_down"], cfg.rms_eps, e2_raw=W["embed"][prev2])
        elif cfg.approx == "linear":
            O.linear_approximator(self.H[hid], W["embed"][prev], W["norm_h"], W["norm_e"], W["w_lin"], cfg.rms_eps)
        else:
            O.ar_approximator(self.H[hid], W["embed"][prev], W["norm_h"], W["norm_e"], W["w_gate"], W["w_up"],
                              W["w_down"], cfg.rms_eps)
        t_mlp = time.perf_counter() - t0
        t0 = time.perf_counter()
        O.draft_sequence(self.H, root, 0, W, M=cfg.M, K2=cfg.K2, B=cfg.B, temperature=cfg.temperature,
                         eps=cfg.rms_eps, mode=cfg.mode, approx=cfg.approx, root_prev=rprev)
        t = time.perf_counter() - t0
        full = t_mlp + max(t - t_mlp, 0.0) * cfg.V / Vs
        return t, full, Vs


def oracle_sample_child(path: str) -> None:
    """Child side of oracle_single_thread: load the sample's tensors, run the oracle once on
    them and print (seconds, estimated seconds per tree, vocabulary used) as JSON."""
    import torch
    import synth
    d = torch.load(path)
    cfg = synth.get_config(d["workload"])
    orc = OracleSample(cfg, d["inp"])
    t, full, Vs = orc.run(d["inp"]["lm_head"].shape[0] / cfg.V)
    print(json.dumps({"t": t, "full": full, "Vs": Vs}), flush=True)


def oracle_single_thread(cfg, inp, frac):
    """The oracle's sample on one host core: a child process started with the BLAS and OpenMP
    thread counts set to 1 before numpy loads (they cannot be changed afterwards). It gets the
    sample's tensors in their own dtype (the vocabulary-dependent ones cut to the sample's
    vocabulary; every token the sample can reach lies below it) through a temporary file."""
    import tempfile
    import torch
    Vs = max(cfg.K2 + cfg.M, int(math.ceil(cfg.V * frac)))
    keys = ("hidden", "root_tok", "root_prev", "norm_h", "norm_e", "w_gate", "w_up", "w_down", "w_lin")
    sample = {k: inp[k][:1] if k in ("hidden", "root_tok", "root_prev") else inp[k]
              for k in keys if inp.get(k) is not None}
    sample["lm_head"] = inp["lm_head"][:Vs].clone()
    sample["embed"] = inp["embed"][:Vs].clone()
    with tempfile.TemporaryDirectory() as td:
        path = os.path.join(td, "sample.pt")
        torch.save({"workload": cfg.name, "inp": sample}, path)
        env = dict(os.environ, OPENBLAS_NUM_THREADS="1", OMP_NUM_THREADS="1", MKL_NUM_THREADS="1")
        r = subprocess.run([sys.executable, os.path.abspath(__file__), "--cpu-sample", path], env=env,
                           capture_output=True, text=True, timeout=900)
    if r.returncode != 0:
        return {"error": (r.stderr.strip().splitlines() or ["child failed"])[-1][:200]}
    res = json.loads(r.stdout.strip().splitlines()[-1])
    return {"value": 1.0 / res["full"], "unit": "trees/s", "cores": 1, "kind": "oracle",
            "sample": f"fp64 numpy oracle on one core, 1 sequence, vocabulary cut to {res['Vs']} of {cfg.V} "
                      f"({res['t']:.1f} s), LM-head/softmax/sort time scaled to the full V"}


def cpu_model() -> str:
    """The host CPU's model name (x86 "model name"; on Arm the implementer / part codes)."""
    try:
        info = open("/proc/cpuinfo").read().splitlines()
    except OSError:
        info = []
    for key in ("model name", "Model name"):
        for line in info:
            if line.startswith(key):
                return line.split(":", 1)[1].strip()
    fields = {}
    for line in info:
        if ":" in line:
            k, v = (x.strip() for x in line.split(":", 1))
            fields.setdefault(k, v)
    if "CPU part" in fields:
        return f"Arm implementer {fields.get('CPU implementer', '?')} part {fields['CPU part']}"
    import platform
    return platform.machine()


def cpu_threads():
    for k in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS"):
        if os.environ.get(k, "").isdigit():
            return int(os.environ[k])
    return os.cpu_count() or 1


# ------------------------------------------------------------------------------ arms

def run_reference(args):
    rank, world, _ = dist_env()
    if world > 1:
        init_dist("gloo")
        if rank != 0:
            return
    import synth
    cfg = synth.get_config(args.workload)
    inp = synth.make_inputs(cfg)
    orc = OracleSample(cfg, inp)
    # calibrate on 1/64 of the vocabulary, then size every step so the run stays ~2 minutes
    _, full_est, _ = orc.run(1 / 64)
    n = max(1, args.steps + args.warmup)
    frac = min(1.0, max(1 / 256, 120.0 / (n * max(full_est, 1e-3))))
    for _ in range(args.warmup):
        orc.run(frac)
    ests = []
    for _ in range(max(1, args.steps)):
        _, full, Vs = orc.run(frac)
        ests.append(full)
    t_tree = sum(ests) / len(ests)
    value = 1.0 / t_tree
    cores = cpu_threads()
    sample = f"fp64 oracle, 1 sequence, vocabulary cut to {Vs} of {cfg.V} per step; time scaled to the full V"
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "trees/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": t_tree * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": cfg.name, "batch": cfg.batch, "d": cfg.d, "V": cfg.V, "I": cfg.I,
                       "gamma": cfg.gamma, "M": cfg.M, "K2": cfg.K2, "B": cfg.B, "approx": cfg.approx},
            "cpu_baseline": {"value": value, "unit": "trees/s", "cores": cores, "cpu_model": cpu_model(),
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": "trees/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def run_gpu(args):
    import torch
    rank, world, local = dist_env()
    if world > 1:
        init_dist("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    import synth
    import paper_2606_03819_gb300 as tf
    from paper_2606_03819_gb300 import binding as Bn

    cfg = synth.get_config(args.workload, seed=rank)
    inp = synth.make_inputs(cfg)
    d = {k: v.to(dev) for k, v in inp.items() if isinstance(v, torch.Tensor)}
    # the two-previous-token approximator takes (x_t, x_{t-1}) per sequence in root_tok
    root_in = inp["root_tok"] if "root_prev" not in inp else \
        torch.stack([inp["root_tok"], inp["root_prev"]], dim=1).contiguous()
    d["root_tok"] = root_in.to(dev)
    dims = Bn.Dims.from_config(cfg)
    dr = tf.Drafter(dims, d, dev)
    hp = Bn.tf_workspace_h_prime(dims, dr.ws)
    H = d["hidden"]
    n1, n2 = cfg.batch * cfg.gamma, cfg.batch * cfg.R
    stream = torch.cuda.current_stream(dev)

    def step():
        # one whole draft-tree build through the public calls: tf_stage1_marginals,
        # tf_stage2_ar_approx, tf_build_tree, tf_tree_mask
        dr.draft(H, d["root_tok"], d["root_pos"])

    def step_timed(ev):
        # the same kernels issued as their pieces, with CUDA events around the two LM-head passes
        Bn.tf_status_reset(dr.ws)
        ev[0].record(stream)
        Bn.tf_lmhead_partials(dims, d["lm_head"], H, n1, dr.ws)
        ev[1].record(stream)
        Bn.tf_lmhead_merge(dims, d["lm_head"], H, n1, dims.K1, dr.top_ids, dr.top_logp, dr.ws)
        Bn.tf_ar_approx(dims, d, H, d["root_tok"], dr.top_ids, None, dr.ws)
        ev[2].record(stream)
        Bn.tf_lmhead_partials(dims, d["lm_head"], hp, n2, dr.ws)
        ev[3].record(stream)
        Bn.tf_lmhead_merge(dims, d["lm_head"], hp, n2, dims.K2, dr.child_ids, dr.child_logp, dr.ws)
        dr.build(d["root_tok"], d["root_pos"])

    for _ in range(max(args.warmup, 3)):
        step()
    torch.cuda.synchronize(dev)
    flags = Bn.tf_status_read(dr.ws)
    # sanity: the pieces give the composite calls' result
    ref = {k: v.clone() for k, v in dr.draft(H, d["root_tok"], d["root_pos"]).items() if v is not None}
    step_timed([torch.cuda.Event(enable_timing=True) for _ in range(4)])
    torch.cuda.synchronize(dev)
    for k in ("node_tok", "node_parent", "mask"):
        assert torch.equal(ref[k], getattr(dr, k)), k

    # ---- the timed region: K whole steps, nothing else on the stream
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    barrier(world, dev)
    torch.cuda.synchronize(dev)
    launches0 = Bn.tf_kernel_launches()
    with ClockSampler(local) as clk:
        t_start.record(stream)
        for i in range(args.steps):
            step()
        t_end.record(stream)
        torch.cuda.synchronize(dev)
    gpu_launches = Bn.tf_kernel_launches() - launches0
    barrier(world, dev)
    elapsed_ms = t_start.elapsed_time(t_end)
    elapsed_ms = max_over_ranks(elapsed_ms, world, dev)
    flags |= Bn.tf_status_read(dr.ws)

    # ---- the LM-head passes timed on their own: the same steps with CUDA events around the two
    #      LM-head launches (an event between two kernels stops the next one from starting early,
    #      so these steps are slightly slower and are not part of `value`)
    n_inst = max(1, min(args.steps, 200))
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(n_inst)]
    i_start = torch.cuda.Event(enable_timing=True)
    i_end = torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize(dev)
    i_start.record(stream)
    for i in range(n_inst):
        step_timed(evs[i])
    i_end.record(stream)
    torch.cuda.synchronize(dev)
    inst_ms_per_step = i_start.elapsed_time(i_end) / n_inst
    lm1 = [e[0].elapsed_time(e[1]) for e in evs]
    lm2 = [e[2].elapsed_time(e[3]) for e in evs]

    trees = cfg.batch * args.steps * world
    value = trees / (elapsed_ms / 1e3)
    ms_per_step = elapsed_ms / args.steps
    peak, peak_kind = peaks()
    step_bytes, lm_bytes = algorithmic_bytes(cfg)
    timing = (f"CUDA events around each LM-head launch over {n_inst} further steps "
              f"({inst_ms_per_step * 1e3:.1f} us per step with the events)")
    roofline = lmhead_roofline(cfg, n1, n2, statistics.mean(lm1), statistics.mean(lm2), (peak, peak_kind),
                               tensor_peak(), profiled_traffic(cfg.name), timing)

    # ---- end to end through the host-buffer entry point
    e2e = None
    if args.e2e_steps > 0:
        n = cfg.B + 1
        pin = lambda t: t.pin_memory()
        h_hidden, h_root, h_pos = pin(inp["hidden"]), pin(root_in), pin(inp["root_pos"])
        outs = dict(node_tok=torch.empty(cfg.batch, n, dtype=torch.int32),
                    node_parent=torch.empty(cfg.batch, n, dtype=torch.int32),
                    node_depth=torch.empty(cfg.batch, n, dtype=torch.int32),
                    node_score=torch.empty(cfg.batch, n, dtype=torch.float32),
                    mask=torch.empty(cfg.batch, n, n, dtype=torch.uint8),
                    pos_ids=torch.empty(cfg.batch, n, dtype=torch.int32),
                    dev_status=torch.empty(cfg.batch, dtype=torch.int32))
        outs = {k: pin(v) for k, v in outs.items()}

        e2e_stream = torch.cuda.Stream(dev)

        def host_step():
            return Bn.tf_draft_tree_host(dims, d, h_hidden, h_root, h_pos, outs["node_tok"], outs["node_parent"],
                                         outs["node_depth"], outs["node_score"], outs["mask"], outs["pos_ids"],
                                         outs["dev_status"], dr.ws, stream=e2e_stream)
        for _ in range(3):
            host_step()
        barrier(world, dev)
        t0 = time.perf_counter()
        for _ in range(args.e2e_steps):
            host_step()
        t_e2e = max_over_ranks(time.perf_counter() - t0, world, dev)
        assert torch.equal(outs["node_tok"], ref["node_tok"].cpu())
        h2d = sum(t.numel() * t.element_size() for t in (h_hidden, h_root, h_pos))
        d2h = sum(t.numel() * t.element_size() for t in outs.values())
        e2e = {"value": cfg.batch * args.e2e_steps * world / t_e2e, "unit": "trees/s",
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h}

    # ---- the same step with torch library calls (rank 0, N = 1; SwiGLU TreeFlash mode only)
    eager = None
    if rank == 0 and world == 1 and args.torch_eager_steps > 0 and cfg.mode == "ar" and cfg.approx == "swiglu":
        try:
            eager = time_torch_eager(cfg, d, H, d["root_tok"], args.torch_eager_steps)
        except Exception as exc:   # a reference point must not cost the measured line
            eager = {"error": f"{type(exc).__name__}: {exc}"[:200]}

    # ---- CPU baseline: the oracle on the host cores (rank 0, N = 1 only)
    cpu = None
    if rank == 0 and world == 1 and args.cpu_baseline_s > 0:
        orc = OracleSample(cfg, inp)
        _, full_est, _ = orc.run(1 / 64)
        frac = min(1.0, max(1 / 64, args.cpu_baseline_s / max(full_est, 1e-3)))
        t, full, Vs = orc.run(frac)
        cpu = {"value": 1.0 / full, "unit": "trees/s", "cores": cpu_threads(), "cpu_model": cpu_model(),
               "kind": "oracle",
               "sample": f"fp64 numpy oracle, 1 sequence, vocabulary cut to {Vs} of {cfg.V} "
                         f"({t:.1f} s), LM-head/softmax/sort time scaled to the full V"}
        # the same oracle on one core, on a smaller cut of the vocabulary (about as long)
        cpu["single_thread"] = oracle_single_thread(cfg, inp, max(1 / 1024, frac / max(cpu_threads(), 1)))

    if rank != 0:
        return
    clocks = clk.summary()
    line = {
        "metric": METRIC, "value": value, "unit": "trees/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "us_per_tree": ms_per_step * 1e3 / cfg.batch,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": cfg.dtype,
        "data": "synthetic (seeded N(0,0.02) weights, hidden states scaled to 2-4 nat marginals)",
        "config": {"workload": cfg.name, "batch": cfg.batch, "d": cfg.d, "V": cfg.V, "I": cfg.I,
                   "gamma": cfg.gamma, "M": cfg.M, "K2": cfg.K2, "B": cfg.B, "R": cfg.R, "approx": cfg.approx,
                   "l2": f"no flush: inputs larger than L2 (W_lm {lm_bytes / 1e9:.3f} GB streamed twice per step)",
                   "parallelism": f"replicas x{world}"},
        "step_roofline": {"algorithmic_bytes": step_bytes, "achieved_gbs": step_bytes / (ms_per_step / 1e3) / 1e9,
                          "peak_gbs": peak, "frac": step_bytes / (ms_per_step / 1e3) / 1e9 / peak,
                          "peak_kind": peak_kind, "nominal_gbs": NOMINAL_HBM_GBS,
                          "frac_nominal": step_bytes / (ms_per_step / 1e3) / 1e9 / NOMINAL_HBM_GBS,
                          "target": "70 % of the HBM roofline, stated against the measured copy rate "
                                    "(peak_gbs); frac_nominal is the same figure against 8 TB/s"},
        "roofline": roofline,
        "clocks": clocks, "e2e": e2e, "gpu_launches": gpu_launches,
        "cpu_baseline": cpu, "torch_eager": eager, "device_flags": flags,
    }
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default=WORKLOAD,
                    help="synthetic workload (synth.CONFIGS); default the measured Qwen3-8B-shape B=64 step")
    ap.add_argument("--e2e-steps", type=int, default=300)
    ap.add_argument("--torch-eager-steps", type=int, default=20,
                    help="steps of the torch library-call reference point (0 = skip)")
    ap.add_argument("--cpu-baseline-s", type=float, default=20.0,
                    help="approximate seconds of oracle work for the cpu_baseline sample (0 = skip)")
    ap.add_argument("--cpu-sample", default=None, help=argparse.SUPPRESS)   # child of oracle_single_thread
    args = ap.parse_args()
    if args.cpu_sample:
        oracle_sample_child(args.cpu_sample)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
