"""The allocation-free LM-head argmax (oos_lm_head_argmax_static), through
the C ABI, against the CPU checker's LM head and against the LM head of
oos_tree_verify_debug on the same rows.

The entry point is for callers that cannot allocate device memory (inside a
CUDA graph that someone else is capturing, under a memory pool they do not
own, with a locked allocator): its scratch is a fixed device array inside the
library that every call shares.  So it is called twice in a row, to check
that the second call starts from a clean state.  The file is collected last on
purpose: it shares nothing with the other tests and must pass both alone in a
fresh process and after them.
"""

import numpy as np
import pytest
import torch

import oracle
from cases import build_case
from gpu_util import GATE, TOL, gpu_cache, gpu_model, max_rel_err, run

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a GPU", allow_module_level=True)

from paper_2608_00814_gb300 import binding as B  # noqa: E402


@pytest.mark.parametrize("name,T", [("tiny", 8), ("mini-bf16", 16), ("mini-bf16", 128)])
def test_static_argmax_matches_oracle_and_verify(name, T):
    case = build_case(name, 0, T=T, plant=3, recipe=dict(kind="uniform", max_depth=6))
    model, w = gpu_model(case)
    kv = gpu_cache(case, case.ctx_len + T)
    g = run(model, kv, case.ctx_len, case.tokens, case.parent)
    hidden = g["debug_outs"].final_hidden     # fp32 [T, H] final-RMSNorm rows from the verify
    # the checker's LM head on the very same rows, in fp64 over the same weights
    ref_arg, ref_t1, ref_t2 = oracle.lm_head_argmax(case.view, hidden.cpu().numpy().astype(np.float64))
    ref_margin = ref_t1 - ref_t2
    dtype = B.OOS_DTYPE_BF16 if case.cfg.dtype == "bf16" else B.OOS_DTYPE_F32
    tol_v, gate_v = TOL[case.cfg.dtype], GATE[case.cfg.dtype]
    for call in range(2):
        arg = torch.full((T,), -7, dtype=torch.int32, device="cuda")
        t1 = torch.full((T,), float("nan"), dtype=torch.float32, device="cuda")
        t2 = torch.full((T,), float("nan"), dtype=torch.float32, device="cuda")
        B.oos_lm_head_argmax_static(dtype, case.cfg.vocab, case.cfg.hidden, w["lm_head"], hidden, T, arg, t1, t2)
        torch.cuda.synchronize()
        a = arg.cpu().numpy()
        v1 = t1.cpu().numpy().astype(np.float64)
        v2 = t2.cpu().numpy().astype(np.float64)
        # vs the checker: fp32 dot products of fp32 rows, so the fp32 tolerance and gate
        assert max_rel_err(v1, ref_t1) <= TOL["f32"], (call, max_rel_err(v1, ref_t1))
        assert max_rel_err(v2, ref_t2) <= TOL["f32"], (call, max_rel_err(v2, ref_t2))
        sep = ref_margin > GATE["f32"]
        assert np.array_equal(a[sep], ref_arg[sep]), call
        assert sep.sum() >= T // 2
        # vs the existing entry point (the verify's fused LM head), at the tolerance of its dtype
        assert max_rel_err(v1, g["top1"].astype(np.float64)) <= tol_v
        assert max_rel_err(v2, g["top2"].astype(np.float64)) <= tol_v
        sep_v = g["top1"] - g["top2"] > gate_v
        assert np.array_equal(a[sep_v], g["argmax"][sep_v]), call


def test_static_argmax_rejects_oversized_T():
    x = torch.zeros(1, dtype=torch.float32, device="cuda")   # never read: the call is rejected first
    i = torch.zeros(1, dtype=torch.int32, device="cuda")
    with pytest.raises(B.OosError) as e:
        B.oos_lm_head_argmax_static(B.OOS_DTYPE_F32, 16, 4, x, x, 129, i, x, x)
    assert e.value.code == B.OOS_EINVAL
