"""GB300 (sm_103a) tree-verification step of OoO-Spec (arXiv 2608.00814).

The verify step -- one forward pass of the target over a packed candidate
tree with an ancestor mask, greedy longest-prefix acceptance, and KV
compaction -- runs entirely in the CUDA library built from csrc/ (C ABI in
include/oos.h).  `binding` marshals PyTorch tensors into that ABI.
"""

from . import binding  # noqa: F401
from .binding import (KVCache, OosError, OosModel, VerifyOutputs, oos_accept_walk,  # noqa: F401
                      oos_kv_compact, oos_last_status, oos_status_string, oos_tree_verify,
                      oos_tree_verify_debug, oos_workspace_bytes, tree_verify)
