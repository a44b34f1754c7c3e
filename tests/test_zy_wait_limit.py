"""The failure path of the device waits, exercised without a fault: a wait
limit of one nanosecond makes the pipeline waits of the verify step give up.
Every kernel then records OOS_ETIMEOUT, drains its own copies and MMAs, frees
its tensor memory and returns; the step reports no accepted path; and a fresh
handle (and the same one with the default limit) verifies correctly again.
Collected near the end: it shares nothing with the other tests."""

import pytest
import torch

import oracle
from cases import build_case
from gpu_util import check_case, check_compaction, gpu_cache, gpu_model, run

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a GPU", allow_module_level=True)

from paper_2608_00814_gb300 import binding as B  # noqa: E402


@pytest.mark.parametrize("name", ["mini-bf16", "tiny"])
def test_wait_limit_runs_out_and_handles_recover(name):
    case = build_case(name, 2)
    model, w = gpu_model(case)
    kv = gpu_cache(case, case.ctx_len + len(case.tokens))
    tok = torch.as_tensor(case.tokens, device="cuda")
    par = torch.as_tensor(case.parent, device="cuda")
    B.oos_set_wait_limit(model, 1)
    outs = B.tree_verify(model, kv, case.ctx_len, tok, par)
    torch.cuda.synchronize()   # the kernels returned
    status = B.oos_last_status(model)
    if case.cfg.dtype == "bf16":
        assert status == B.OOS_ETIMEOUT
        assert int(outs.accepted_len.item()) == 0 and int(outs.bonus.item()) == -1
    else:
        # the fp32 CUDA-core path has no pipeline waits: the limit changes nothing
        assert status == B.OOS_OK
    # the same handle with the default limit, and a fresh handle, verify correctly
    B.oos_set_wait_limit(model, 0)
    r = oracle.verify_tree(case.view, case.cache_k64, case.cache_v64, case.ctx_len, case.tokens, case.parent)
    g = run(model, kv, case.ctx_len, case.tokens, case.parent)
    check_case(case, g, r)
    fresh = B.OosModel(case.cfg, w)
    kv2 = gpu_cache(case, case.ctx_len + len(case.tokens))
    g2 = run(fresh, kv2, case.ctx_len, case.tokens, case.parent)
    check_case(case, g2, r)
    check_compaction(fresh, kv2, case.ctx_len, g2)
