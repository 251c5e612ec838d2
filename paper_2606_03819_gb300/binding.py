"""ctypes binding of the TreeFlash C ABI (include/treeflash.h).

Argument marshalling only: every function here passes raw device pointers of torch tensors,
the current CUDA stream and the dims/weights structs to the function of the same name in
lib/libtreeflash.so and raises TreeFlashError if it returns a status other than TF_OK. All
computation happens in the library's CUDA kernels; nothing here computes any part of the
path, and there is no fallback: without the built library every call raises.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass
from typing import Optional

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "lib", "libtreeflash.so")

TF_OK, TF_ERR_INVALID_ARG, TF_ERR_UNSUPPORTED, TF_ERR_WORKSPACE, TF_ERR_CUDA, TF_ERR_DEVICE_STATUS, \
    TF_ERR_TIMEOUT = range(7)
TF_BF16, TF_F32 = 0, 1
MODES = {"ar": 0, "marginal": 1, "marginal_mary": 2}
APPROX = {"swiglu": 0, "linear": 1, "swiglu_2prev": 2}
TF_DEV_BAD_TOKEN, TF_DEV_UNDERFULL, TF_DEV_NONFINITE, TF_DEV_TIMEOUT, TF_DEV_RECOMPUTED = 1, 2, 4, 8, 16


class TreeFlashError(RuntimeError):
    def __init__(self, fn: str, status: int, msg: str):
        super().__init__(f"{fn}: {msg} (status {status})")
        self.status = status


class TfDims(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("d", ctypes.c_int32), ("V", ctypes.c_int32),
                ("I", ctypes.c_int32), ("gamma", ctypes.c_int32), ("M", ctypes.c_int32),
                ("K2", ctypes.c_int32), ("B", ctypes.c_int32), ("temperature", ctypes.c_float),
                ("rms_eps", ctypes.c_float), ("dtype", ctypes.c_int32), ("mode", ctypes.c_int32),
                ("approx", ctypes.c_int32)]


class TfWeights(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in
                ("lm_head", "embed", "norm_h", "norm_e", "w_gate", "w_up", "w_down", "w_lin")]


EXPORTS = ("tf_status_string", "tf_version", "tf_kernel_launches", "tf_workspace_size", "tf_status_reset", "tf_status_read",
           "tf_stage1_marginals", "tf_stage2_ar_approx", "tf_build_tree", "tf_tree_mask", "tf_build_tree_mask",
           "tf_draft_tree_host", "tf_lmhead_partials", "tf_lmhead_merge", "tf_ar_approx",
           "tf_workspace_h_prime", "tf_workspace_view", "tf_stage1_marginals_static", "tf_accept_walk",
           "tf_set_wait_limit_ns")

_lib = None


def load_library(path: Optional[str] = None) -> ctypes.CDLL:
    """Load lib/libtreeflash.so (built by __graft_entry__.build()). Raises if it is missing."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = path or LIB_PATH
    if not os.path.exists(p):
        raise RuntimeError(f"TreeFlash CUDA library not found at {p}; build it with "
                           "`python -c 'import __graft_entry__ as g; g.build()'`")
    lib = ctypes.CDLL(p)
    P, I32, SZ = ctypes.c_void_p, ctypes.c_int32, ctypes.c_size_t
    D, W = ctypes.POINTER(TfDims), ctypes.POINTER(TfWeights)
    sig = {
        "tf_status_string": (ctypes.c_char_p, [ctypes.c_int]),
        "tf_version": (I32, []),
        "tf_kernel_launches": (ctypes.c_uint64, []),
        "tf_set_wait_limit_ns": (ctypes.c_int, [ctypes.c_uint64]),
        "tf_workspace_size": (ctypes.c_int, [D, ctypes.POINTER(SZ)]),
        "tf_status_reset": (ctypes.c_int, [P, SZ, P]),
        "tf_status_read": (ctypes.c_int, [P, SZ, ctypes.POINTER(I32), P]),
        "tf_stage1_marginals": (ctypes.c_int, [D, W, P, P, P, P, SZ, P]),
        "tf_stage2_ar_approx": (ctypes.c_int, [D, W, P, P, P, P, P, P, SZ, P]),
        "tf_build_tree": (ctypes.c_int, [D, P, P, P, P, P, P, P, P, P, P, P]),
        "tf_tree_mask": (ctypes.c_int, [D, P, P, P, P, P, P]),
        "tf_build_tree_mask": (ctypes.c_int, [D, P, P, P, P, P, P, P, P, P, P, P, P, P, P]),
        "tf_draft_tree_host": (ctypes.c_int, [D, W, P, P, P, P, P, P, P, P, P, P, P, SZ, P]),
        "tf_lmhead_partials": (ctypes.c_int, [D, P, P, I32, P, SZ, P]),
        "tf_lmhead_merge": (ctypes.c_int, [D, P, P, I32, I32, P, P, P, SZ, P]),
        "tf_ar_approx": (ctypes.c_int, [D, W, P, P, P, P, P, SZ, P]),
        "tf_workspace_h_prime": (ctypes.c_int, [D, P, SZ, ctypes.POINTER(P)]),
        "tf_workspace_view": (ctypes.c_int, [D, P, SZ, I32, ctypes.POINTER(P), ctypes.POINTER(SZ)]),
        "tf_stage1_marginals_static": (ctypes.c_int, [D, W, P, P, P, P, P]),
        "tf_accept_walk": (ctypes.c_int, [D, P, P, P, P, P, P, P]),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype, f.argtypes = res, args
    if path is None:
        _lib = lib
    return lib


def _check(fn: str, status: int):
    if status != TF_OK:
        msg = load_library().tf_status_string(status).decode()
        raise TreeFlashError(fn, status, msg)


@dataclass(frozen=True)
class Dims:
    batch: int
    d: int
    V: int
    I: int
    gamma: int
    M: int
    K2: int
    B: int
    temperature: float = 1.0
    rms_eps: float = 1e-6
    dtype: str = "bf16"
    mode: str = "ar"
    approx: str = "swiglu"      # "swiglu" (Eq. 1); the ablations' "linear" and "swiglu_2prev"

    @property
    def R(self) -> int:
        if self.approx == "swiglu_2prev" and self.mode == "ar":
            return 1 if self.gamma == 1 else 1 + self.M + self.M * self.M * (self.gamma - 2)
        return 1 + self.M * (self.gamma - 1)

    @property
    def K1(self) -> int:
        return max(self.M, self.K2)

    @property
    def k_in(self) -> int:
        """Width of the approximator input x: 2d, or 3d with two previous tokens."""
        return (3 if self.approx == "swiglu_2prev" and self.mode == "ar" else 2) * self.d

    @property
    def torch_dtype(self):
        return torch.bfloat16 if self.dtype == "bf16" else torch.float32

    def c(self) -> TfDims:
        return TfDims(self.batch, self.d, self.V, self.I, self.gamma, self.M, self.K2, self.B,
                      self.temperature, self.rms_eps, TF_BF16 if self.dtype == "bf16" else TF_F32,
                      MODES[self.mode], APPROX[self.approx])

    @classmethod
    def from_config(cls, cfg) -> "Dims":
        return cls(cfg.batch, cfg.d, cfg.V, cfg.I, cfg.gamma, cfg.M, cfg.K2, cfg.B, cfg.temperature,
                   cfg.rms_eps, cfg.dtype, cfg.mode, getattr(cfg, "approx", "swiglu"))


WEIGHT_KEYS = ("lm_head", "embed", "norm_h", "norm_e", "w_gate", "w_up", "w_down", "w_lin")


def _ptr(t: Optional[torch.Tensor]):
    if t is None:
        return None
    if not t.is_contiguous():
        raise ValueError("tensors passed to the TreeFlash ABI must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def weights_struct(w: dict) -> TfWeights:
    return TfWeights(*[w[k].data_ptr() if w.get(k) is not None else None for k in WEIGHT_KEYS])


def tf_version() -> int:
    return load_library().tf_version()


def tf_kernel_launches() -> int:
    """Kernels launched by the library so far in this process."""
    return int(load_library().tf_kernel_launches())


def tf_set_wait_limit_ns(ns: int) -> None:
    """Limit of the tensor-core kernels' waits for progress, for every later launch (0 = the
    default 2 s); a limit below a copy's latency makes calls time out (TF_DEV_TIMEOUT)."""
    _check("tf_set_wait_limit_ns", load_library().tf_set_wait_limit_ns(int(ns)))


def tf_workspace_size(dims: Dims) -> int:
    n = ctypes.c_size_t(0)
    _check("tf_workspace_size", load_library().tf_workspace_size(ctypes.byref(dims.c()), ctypes.byref(n)))
    return n.value


def alloc_workspace(dims: Dims, device="cuda") -> torch.Tensor:
    """A torch-owned workspace (256-byte aligned) of tf_workspace_size bytes."""
    n = tf_workspace_size(dims)
    buf = torch.empty(n + 256, dtype=torch.uint8, device=device)
    off = (-buf.data_ptr()) % 256
    return buf[off:off + n]


def tf_status_reset(ws: torch.Tensor, stream=None):
    _check("tf_status_reset", load_library().tf_status_reset(_ptr(ws), ws.numel(), _stream(stream)))


def tf_status_read(ws: torch.Tensor, stream=None, raise_on_error: bool = False) -> int:
    flags = ctypes.c_int32(0)
    st = load_library().tf_status_read(_ptr(ws), ws.numel(), ctypes.byref(flags), _stream(stream))
    if st == TF_ERR_CUDA or raise_on_error:
        _check("tf_status_read", st)
    return flags.value


def tf_stage1_marginals(dims: Dims, w: dict, hidden, top_ids, top_logp, ws, stream=None):
    _check("tf_stage1_marginals", load_library().tf_stage1_marginals(
        ctypes.byref(dims.c()), ctypes.byref(weights_struct(w)), _ptr(hidden), _ptr(top_ids),
        _ptr(top_logp), _ptr(ws), ws.numel(), _stream(stream)))


def tf_stage2_ar_approx(dims: Dims, w: dict, hidden, root_tok, top_ids, child_ids, child_logp, ws,
                        stream=None):
    _check("tf_stage2_ar_approx", load_library().tf_stage2_ar_approx(
        ctypes.byref(dims.c()), ctypes.byref(weights_struct(w)), _ptr(hidden), _ptr(root_tok),
        _ptr(top_ids), _ptr(child_ids), _ptr(child_logp), _ptr(ws), ws.numel(), _stream(stream)))


def tf_build_tree(dims: Dims, root_tok, top_ids, top_logp, child_ids, child_logp, node_tok, node_parent,
                  node_depth, node_score, dev_status, stream=None):
    _check("tf_build_tree", load_library().tf_build_tree(
        ctypes.byref(dims.c()), _ptr(root_tok), _ptr(top_ids), _ptr(top_logp), _ptr(child_ids),
        _ptr(child_logp), _ptr(node_tok), _ptr(node_parent), _ptr(node_depth), _ptr(node_score),
        _ptr(dev_status), _stream(stream)))


def tf_tree_mask(dims: Dims, node_parent, node_depth, root_pos, mask, pos_ids, stream=None):
    _check("tf_tree_mask", load_library().tf_tree_mask(
        ctypes.byref(dims.c()), _ptr(node_parent), _ptr(node_depth), _ptr(root_pos), _ptr(mask),
        _ptr(pos_ids), _stream(stream)))


def tf_build_tree_mask(dims: Dims, root_tok, root_pos, top_ids, top_logp, child_ids, child_logp, node_tok,
                       node_parent, node_depth, node_score, mask, pos_ids, dev_status, stream=None):
    _check("tf_build_tree_mask", load_library().tf_build_tree_mask(
        ctypes.byref(dims.c()), _ptr(root_tok), _ptr(root_pos), _ptr(top_ids), _ptr(top_logp), _ptr(child_ids),
        _ptr(child_logp), _ptr(node_tok), _ptr(node_parent), _ptr(node_depth), _ptr(node_score), _ptr(mask),
        _ptr(pos_ids), _ptr(dev_status), _stream(stream)))


def tf_draft_tree_host(dims: Dims, w: dict, hidden, root_tok, root_pos, node_tok, node_parent, node_depth,
                       node_score, mask, pos_ids, dev_status, ws, stream=None):
    """Host tensors in and out (pinned memory recommended); weights and workspace on the device."""
    st = load_library().tf_draft_tree_host(
        ctypes.byref(dims.c()), ctypes.byref(weights_struct(w)), _ptr(hidden), _ptr(root_tok),
        _ptr(root_pos), _ptr(node_tok), _ptr(node_parent), _ptr(node_depth), _ptr(node_score), _ptr(mask),
        _ptr(pos_ids), _ptr(dev_status), _ptr(ws), ws.numel(), _stream(stream))
    if st not in (TF_OK, TF_ERR_DEVICE_STATUS):
        _check("tf_draft_tree_host", st)
    return st


def tf_accept_walk(dims: Dims, node_tok, node_parent, verifier_tok, accept_len, accept_path, next_tok,
                   stream=None):
    _check("tf_accept_walk", load_library().tf_accept_walk(
        ctypes.byref(dims.c()), _ptr(node_tok), _ptr(node_parent), _ptr(verifier_tok), _ptr(accept_len),
        _ptr(accept_path), _ptr(next_tok), _stream(stream)))


def tf_lmhead_partials(dims: Dims, lm_head, x, n_rows: int, ws, stream=None):
    _check("tf_lmhead_partials", load_library().tf_lmhead_partials(
        ctypes.byref(dims.c()), _ptr(lm_head), _ptr(x), n_rows, _ptr(ws), ws.numel(), _stream(stream)))


def tf_lmhead_merge(dims: Dims, lm_head, x, n_rows: int, k: int, out_ids, out_logp, ws, stream=None):
    _check("tf_lmhead_merge", load_library().tf_lmhead_merge(
        ctypes.byref(dims.c()), _ptr(lm_head), _ptr(x), n_rows, k, _ptr(out_ids), _ptr(out_logp), _ptr(ws),
        ws.numel(), _stream(stream)))


def tf_ar_approx(dims: Dims, w: dict, hidden, root_tok, top_ids, h_prime, ws, stream=None):
    _check("tf_ar_approx", load_library().tf_ar_approx(
        ctypes.byref(dims.c()), ctypes.byref(weights_struct(w)), _ptr(hidden), _ptr(root_tok), _ptr(top_ids),
        _ptr(h_prime), _ptr(ws), ws.numel(), _stream(stream)))


def tf_workspace_h_prime(dims: Dims, ws) -> torch.Tensor:
    """h' [b, R, d] as a tensor view of the workspace (no copy)."""
    p = ctypes.c_void_p()
    _check("tf_workspace_h_prime", load_library().tf_workspace_h_prime(
        ctypes.byref(dims.c()), _ptr(ws), ws.numel(), ctypes.byref(p)))
    off = p.value - ws.data_ptr()
    esize = 2 if dims.dtype == "bf16" else 4
    n = dims.batch * dims.R * dims.d * esize
    return ws[off:off + n].view(dims.torch_dtype).view(dims.batch, dims.R, dims.d)


TF_VIEW_X, TF_VIEW_A, TF_VIEW_H_PRIME, TF_VIEW_HALVES, TF_VIEW_CHUNKS = 0, 1, 2, 3, 4


def tf_workspace_view(dims: Dims, ws, view: int, n_rows: Optional[int] = None) -> torch.Tensor:
    """x [b*R, k_in], A [b*R, I] or h' [b*R, d] as a tensor view of the workspace (no copy); for
    TF_VIEW_HALVES / TF_VIEW_CHUNKS the partials of the last LM-head pass over n_rows rows as
    float32 [n_tiles, 2 or 8, n_rows, 4]."""
    p, n = ctypes.c_void_p(), ctypes.c_size_t()
    _check("tf_workspace_view", load_library().tf_workspace_view(
        ctypes.byref(dims.c()), _ptr(ws), ws.numel(), view, ctypes.byref(p), ctypes.byref(n)))
    off = p.value - ws.data_ptr()
    if view in (TF_VIEW_HALVES, TF_VIEW_CHUNKS):
        n_tiles = (dims.V + 255) // 256
        parts = 2 if view == TF_VIEW_HALVES else 8
        nb = n_tiles * parts * n_rows * 16
        return ws[off:off + nb].view(torch.float32).view(n_tiles, parts, n_rows, 4)
    cols = {TF_VIEW_X: dims.k_in, TF_VIEW_A: dims.I, TF_VIEW_H_PRIME: dims.d}[view]
    return ws[off:off + n.value].view(dims.torch_dtype).view(dims.batch * dims.R, cols)


TF_STATIC_SCRATCH_BYTES = 8 << 20


def tf_stage1_marginals_static(dims: Dims, w: dict, hidden, top_ids, top_logp, dev_status, stream=None):
    """tf_stage1_marginals for callers that cannot allocate: no workspace, the library's own fixed
    scratch array instead. dev_status is a 1-element int32 device tensor that receives the call's
    TF_DEV_* flags. Calls that overlap on the GPU share that array and race."""
    _check("tf_stage1_marginals_static", load_library().tf_stage1_marginals_static(
        ctypes.byref(dims.c()), ctypes.byref(weights_struct(w)), _ptr(hidden), _ptr(top_ids),
        _ptr(top_logp), _ptr(dev_status), _stream(stream)))
