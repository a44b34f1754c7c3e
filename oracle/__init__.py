"""CPU checker for the tree-verification step -- TEST INFRASTRUCTURE ONLY.

Only the test suite, `__graft_entry__.smoke()` and the benchmark's CPU-baseline
leg may import it.  The product path never does.
"""

from .tree_verify import (TreeError, accept, attend, cache_format, compact, decode_sequence,  # noqa: F401
                          decode_step, greedy_continuation, kv_format, lm_head_argmax, mlp, prefill,
                          qkv, rms_norm, rope, rope_inv_freq, rope_scaling, silu, tree_structure,
                          verify_and_accept,
                          verify_tree)
