"""TreeFlash drafting hot path on one GB300: Python side of the C ABI in include/treeflash.h.

`binding` exposes every C entry point under its own name (argument marshalling only);
`Drafter` owns the torch-allocated workspace and output buffers of one configuration and runs
the four calls of a drafting step on the current CUDA stream.
"""
from .binding import (Dims, TreeFlashError, alloc_workspace, load_library, tf_ar_approx, tf_build_tree,
                      tf_draft_tree_host, tf_lmhead_merge, tf_lmhead_partials, tf_stage1_marginals,
                      tf_stage2_ar_approx, tf_status_read, tf_status_reset, tf_tree_mask, tf_version,
                      tf_workspace_size)
from .drafter import Drafter

__all__ = ["Dims", "Drafter", "TreeFlashError", "alloc_workspace", "load_library", "tf_ar_approx",
           "tf_build_tree", "tf_draft_tree_host", "tf_lmhead_merge", "tf_lmhead_partials",
           "tf_stage1_marginals", "tf_stage2_ar_approx", "tf_status_read", "tf_status_reset",
           "tf_tree_mask", "tf_version", "tf_workspace_size"]
