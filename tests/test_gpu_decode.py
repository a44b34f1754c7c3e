"""The device decode loop (oos_decode) against the CPU checker's decode loop
(oracle/decode_loop.py) and against plain greedy decoding, through the C ABI.

The loop is lossless (Section 5, "Metrics and Correctness Audit"): whatever
the bank proposes, the committed tokens are the target's greedy continuation.
Exact comparison is meaningful only while the greedy decisions are well
separated (the margin gate), so every check covers the committed tokens up to
the first decision whose top-1/top-2 margin is within the gate.
"""

import numpy as np
import pytest
import torch

import oracle
from cases import build_case, root_token
from gpu_util import GATE, TOL, gpu_cache, gpu_model, max_rel_err, to_f64
from oracle.decode_loop import speculative_decode
from synth import gen
from synth.model import ROOT

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a GPU", allow_module_level=True)

from paper_2608_00814_gb300 import binding as B  # noqa: E402

EOS = 2


def _separated_root(case, n, gate, tries=12):
    """A root of the seeded stream whose first n greedy decisions all clear the
    gate; falls back to the one with the longest separated prefix."""
    roots = gen.uniform_int(gen.tensor_key(1, ROOT), tries, case.cfg.vocab)
    best = None
    for r in roots:
        toks, margins = oracle.greedy_continuation(case.view, case.cache_k64, case.cache_v64, case.ctx_len, int(r), n)
        ok = next((i for i, m in enumerate(margins) if m <= gate), n)
        if best is None or ok > best[0]:
            best = (ok, int(r), toks, margins)
        if ok == n:
            break
    return best


def _bank(seq, vocab, seed, n_views=8):
    """Hint bank: views of `seq` (the root and its greedy continuation), some
    with one token changed, between random tokens, joined by EOS."""
    rng = np.random.default_rng(seed)
    out = []
    for k in range(n_views):
        out += rng.integers(3, vocab, size=int(rng.integers(3, 20))).tolist() + [EOS]
        a = int(rng.integers(0, max(1, len(seq) - 6)))
        b = min(len(seq), a + int(rng.integers(5, 24)))
        view = list(seq[a:b])
        if k % 3 == 1 and len(view) > 4:
            j = int(rng.integers(2, len(view)))
            view[j] = 3 + (view[j] + 7) % (vocab - 3)
        out += view + [EOS]
    return np.asarray(out, np.int32)


@pytest.mark.parametrize("name,n_rounds,max_nodes,overrides", [("tiny", 12, 16, None), ("mini-bf16", 8, 32, None),
                                                                ("mini-bf16", 6, 24, dict(cache_dtype="f16"))])
def test_decode_loop_matches_oracle_and_greedy(name, n_rounds, max_nodes, overrides):
    case = build_case(name, 0, cfg_overrides=overrides)
    cfg = case.cfg
    gate = GATE[cfg.dtype]
    n_ref = n_rounds * max_nodes
    ok, root, ref, margins = _separated_root(case, 24, gate)
    assert ok >= 8, "no root with a well-separated greedy start"
    seq = [root] + [int(t) for t in ref]
    bank = _bank(seq, cfg.vocab, 5)
    depth, max_lanes = 12, 6
    # the CPU checker's loop on the same inputs
    o = speculative_decode(case.view, case.cache_k64, case.cache_v64, case.ctx_len, root, ok, bank.tolist(), EOS,
                           (), max_lanes, depth, max_nodes)
    # the device loop
    model, _ = gpu_model(case, max_T=max_nodes)
    kv = gpu_cache(case, case.ctx_len + n_rounds * max_nodes)
    committed = torch.zeros(1 + n_ref, dtype=torch.int32, device="cuda")
    committed[0] = root
    d_bank = torch.as_tensor(bank, device="cuda")
    mat = torch.full((n_rounds,), -1, dtype=torch.int32, device="cuda")
    state = torch.zeros(3, dtype=torch.int32, device="cuda")
    ws = torch.empty(B.oos_decode_workspace_bytes(int(bank.size)) + 256, dtype=torch.uint8, device="cuda")
    ws_al = ws[(-ws.data_ptr()) % 256:]
    B.oos_decode(model, kv, case.ctx_len, committed, 1, d_bank, EOS, max_lanes, depth, max_nodes, n_rounds, mat, state,
                 ws_al)
    torch.cuda.synchronize()
    assert B.oos_last_status(model) == B.OOS_OK
    st = state.cpu().tolist()
    g_mat = mat.cpu().tolist()
    assert st[2] == n_rounds and all(m >= 1 for m in g_mat)
    n_new = st[1] - 1
    assert n_new == sum(g_mat) and st[0] == case.ctx_len + n_new
    toks = committed.cpu().tolist()[1:1 + n_new]
    # lossless: the committed tokens are the greedy continuation (within the gated prefix)
    k = min(n_new, ok)
    assert toks[:k] == [int(t) for t in ref[:k]]
    assert o["tokens"][:k] == toks[:k]
    # #MAT per call equals the checker's for every round inside the gated prefix
    done = 0
    for r, m in enumerate(g_mat):
        if done + m > ok or r >= len(o["mat"]):
            break
        assert m == o["mat"][r], (r, g_mat, o["mat"])
        done += m
    assert done >= min(ok, 8)
    assert max(g_mat) > 1, "no draft token was ever accepted"
    # the committed cache equals the checker's loop cache (tolerance of the dtype)
    n_cmp = min(done, len(o["cache_k"][0]) - case.ctx_len)
    for l in range(cfg.n_layers):
        for cur, refc in ((kv.k[l], o["cache_k"][l]), (kv.v[l], o["cache_v"][l])):
            g = to_f64(cfg, cur[case.ctx_len:case.ctx_len + n_cmp])
            assert max_rel_err(g, refc[case.ctx_len:case.ctx_len + n_cmp]) <= TOL[cfg.dtype]


def test_decode_loop_without_matches_is_vanilla():
    """A bank that never matches gives trees of the root alone: one token per
    round (#MAT 1, plain decoding) and the greedy tokens."""
    case = build_case("tiny", 1)
    root = root_token(case.cfg, 1)
    ref, margins = oracle.greedy_continuation(case.view, case.cache_k64, case.cache_v64, case.ctx_len, root, 6)
    model, _ = gpu_model(case, max_T=8)
    n_rounds = 6
    kv = gpu_cache(case, case.ctx_len + n_rounds * 8)
    committed = torch.zeros(1 + n_rounds * 8, dtype=torch.int32, device="cuda")
    committed[0] = root
    bank = torch.full((64,), EOS, dtype=torch.int32, device="cuda")   # EOS only: nothing can follow a match
    mat = torch.zeros(n_rounds, dtype=torch.int32, device="cuda")
    state = torch.zeros(3, dtype=torch.int32, device="cuda")
    ws = torch.empty(B.oos_decode_workspace_bytes(64) + 256, dtype=torch.uint8, device="cuda")
    ws_al = ws[(-ws.data_ptr()) % 256:]
    B.oos_decode(model, kv, case.ctx_len, committed, 1, bank, EOS, 4, 8, 8, n_rounds, mat, state, ws_al)
    torch.cuda.synchronize()
    assert mat.cpu().tolist() == [1] * n_rounds
    ok = next((i for i, m in enumerate(margins) if m <= GATE["f32"]), len(margins))
    assert committed.cpu().tolist()[1:1 + ok] == [int(t) for t in ref[:ok]]


def test_decode_loop_host_errors():
    case = build_case("tiny", 0)
    model, _ = gpu_model(case, max_T=8)
    kv = gpu_cache(case, case.ctx_len + 16)
    committed = torch.zeros(64, dtype=torch.int32, device="cuda")
    bank = torch.zeros(16, dtype=torch.int32, device="cuda")
    mat = torch.zeros(4, dtype=torch.int32, device="cuda")
    state = torch.zeros(3, dtype=torch.int32, device="cuda")
    ws = torch.empty(B.oos_decode_workspace_bytes(16) + 256, dtype=torch.uint8, device="cuda")
    ws_al = ws[(-ws.data_ptr()) % 256:]
    with pytest.raises(B.OosError) as e:   # 4 rounds of 8 nodes need 32 slots past ctx
        B.oos_decode(model, kv, case.ctx_len, committed, 1, bank, EOS, 4, 8, 8, 4, mat, state, ws_al)
    assert e.value.code == B.OOS_ECAPACITY
    with pytest.raises(B.OosError) as e:   # node budget above the handle's max_T
        B.oos_decode(model, kv, case.ctx_len, committed, 1, bank, EOS, 4, 8, 9, 1, mat, state, ws_al)
    assert e.value.code == B.OOS_EINVAL
    with pytest.raises(B.OosError) as e:
        B.oos_decode(model, kv, case.ctx_len, committed, 1, bank, EOS, 4, 8, 8, 1, mat, state, ws_al[1:])
    assert e.value.code == B.OOS_EWORKSPACE
