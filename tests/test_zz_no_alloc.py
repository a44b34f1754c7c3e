"""The allocation-free LM-head argmax (oos_lm_head_argmax_static) against the
LM head of oos_tree_verify_debug, through the C ABI.

Collected last on purpose: it shares nothing with the other tests and must
pass both alone in a fresh process and after them.  Its scratch is a fixed
device array inside the library, so it is called twice in a row to check that
the second call starts from a clean state.
"""

import numpy as np
import pytest
import torch

from cases import build_case
from gpu_util import gpu_cache, gpu_model, run

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a GPU", allow_module_level=True)

from paper_2608_00814_gb300 import binding as B  # noqa: E402


@pytest.mark.parametrize("name,T", [("tiny", 8), ("mini-bf16", 16), ("mini-bf16", 128)])
def test_static_argmax_matches_verify_lm_head(name, T):
    case = build_case(name, 0, T=T, plant=3, recipe=dict(kind="uniform", max_depth=6))
    model, w = gpu_model(case)
    kv = gpu_cache(case, case.ctx_len + T)
    g = run(model, kv, case.ctx_len, case.tokens, case.parent)
    hidden = g["outs"].final_hidden            # fp32 [T, H] final-RMSNorm rows from the verify
    dtype = B.OOS_DTYPE_BF16 if case.cfg.dtype == "bf16" else B.OOS_DTYPE_F32
    for call in range(2):
        arg = torch.full((T,), -7, dtype=torch.int32, device="cuda")
        t1 = torch.full((T,), float("nan"), dtype=torch.float32, device="cuda")
        t2 = torch.full((T,), float("nan"), dtype=torch.float32, device="cuda")
        B.oos_lm_head_argmax_static(dtype, case.cfg.vocab, case.cfg.hidden, w["lm_head"], hidden, T, arg, t1, t2)
        torch.cuda.synchronize()
        a, v1, v2 = arg.cpu().numpy(), t1.cpu().numpy(), t2.cpu().numpy()
        # the verify's LM head reads bf16 hi/lo activations; this one reads the fp32 rows: logits agree to ~1e-5
        np.testing.assert_allclose(v1, g["top1"], rtol=0, atol=2e-3)
        np.testing.assert_allclose(v2, g["top2"], rtol=0, atol=2e-3)
        sep = g["top1"] - g["top2"] > 4e-3
        assert np.array_equal(a[sep], g["argmax"][sep]), call
        assert sep.sum() >= T // 2


def test_static_argmax_rejects_oversized_T():
    x = torch.zeros(1, dtype=torch.float32, device="cuda")   # never read: the call is rejected first
    i = torch.zeros(1, dtype=torch.int32, device="cuda")
    with pytest.raises(B.OosError) as e:
        B.oos_lm_head_argmax_static(B.OOS_DTYPE_F32, 16, 4, x, x, 129, i, x, x)
    assert e.value.code == B.OOS_EINVAL
