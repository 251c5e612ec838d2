"""One drafting step (Algorithm 1, both parts, plus the verifier mask) over the C ABI.

The Drafter allocates, once, the workspace and every output tensor with torch on the target
device, then each `draft` call queues tf_stage1_marginals -> tf_stage2_ar_approx (TreeFlash
mode only) -> tf_build_tree_mask (the tree, then its verifier mask) on the current stream.
Returned tensors are views of the Drafter's buffers and are overwritten by the next call.
"""
from __future__ import annotations

import torch

from . import binding as B


class Drafter:
    def __init__(self, dims: B.Dims, weights: dict, device="cuda"):
        B.load_library()
        self.dims = dims
        self.w = {k: weights[k] for k in B.WEIGHT_KEYS if weights.get(k) is not None}
        dev = torch.device(device)
        b, g, n = dims.batch, dims.gamma, dims.B + 1
        i32 = dict(dtype=torch.int32, device=dev)
        f32 = dict(dtype=torch.float32, device=dev)
        self.ws = B.alloc_workspace(dims, dev)
        self.top_ids = torch.empty(b, g, dims.K1, **i32)
        self.top_logp = torch.empty(b, g, dims.K1, **f32)
        ar = dims.mode == "ar"
        self.child_ids = torch.empty(b, dims.R, dims.K2, **i32) if ar else None
        self.child_logp = torch.empty(b, dims.R, dims.K2, **f32) if ar else None
        self.node_tok = torch.empty(b, n, **i32)
        self.node_parent = torch.empty(b, n, **i32)
        self.node_depth = torch.empty(b, n, **i32)
        self.node_score = torch.empty(b, n, **f32)
        self.dev_status = torch.empty(b, **i32)
        self.mask = torch.empty(b, n, n, dtype=torch.uint8, device=dev)
        self.pos_ids = torch.empty(b, n, **i32)

    def stage1(self, hidden, stream=None):
        B.tf_stage1_marginals(self.dims, self.w, hidden, self.top_ids, self.top_logp, self.ws, stream)
        return self.top_ids, self.top_logp

    def stage2(self, hidden, root_tok, stream=None):
        B.tf_stage2_ar_approx(self.dims, self.w, hidden, root_tok, self.top_ids, self.child_ids,
                              self.child_logp, self.ws, stream)
        return self.child_ids, self.child_logp

    def build(self, root_tok, root_pos, stream=None):
        B.tf_build_tree_mask(self.dims, root_tok, root_pos, self.top_ids, self.top_logp, self.child_ids,
                             self.child_logp, self.node_tok, self.node_parent, self.node_depth, self.node_score,
                             self.mask, self.pos_ids, self.dev_status, stream)

    def draft(self, hidden, root_tok, root_pos, stream=None) -> dict:
        self.stage1(hidden, stream)
        if self.dims.mode == "ar":
            self.stage2(hidden, root_tok, stream)
        self.build(root_tok, root_pos, stream)
        return self.outputs()

    def outputs(self) -> dict:
        return dict(top_ids=self.top_ids, top_logp=self.top_logp, child_ids=self.child_ids,
                    child_logp=self.child_logp, node_tok=self.node_tok, node_parent=self.node_parent,
                    node_depth=self.node_depth, node_score=self.node_score, dev_status=self.dev_status,
                    mask=self.mask, pos_ids=self.pos_ids)

    def status(self, stream=None) -> int:
        """Synchronise and return the workspace's TF_DEV_* flags."""
        return B.tf_status_read(self.ws, stream)
