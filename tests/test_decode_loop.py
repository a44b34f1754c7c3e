"""Pins of the multi-step decode loop checker (oracle/decode_loop.py) -- no GPU.

The loop must be lossless: whatever the hint bank proposes, the committed
tokens are the target's greedy autoregressive trajectory (Eq. 1 applied token
by token, computed independently by plain decoding), and the committed cache
is the one plain decoding builds.  #MAT follows from the bank: 1 per call with
nothing to match (vanilla decoding), depth + 1 when the bank holds the greedy
continuation."""

import os
import sys

import numpy as np
import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(HERE))
sys.path.insert(0, HERE)

import oracle  # noqa: E402
from cases import build_case  # noqa: E402
from oracle.decode_loop import speculative_decode  # noqa: E402

EOS = 1


@pytest.fixture(scope="module")
def tiny():
    case = build_case("tiny", 5, plant=0)
    root = int(case.tokens[0])
    greedy, _ = oracle.greedy_continuation(case.view, case.cache_k64, case.cache_v64, case.ctx_len, root, 40)
    return case, root, greedy


def _run(case, root, n, bank, **kw):
    return speculative_decode(case.view, case.cache_k64, case.cache_v64, case.ctx_len, root, n, bank, EOS, **kw)


def test_vanilla_when_nothing_matches(tiny):
    case, root, greedy = tiny
    r = _run(case, root, 12, [EOS, EOS])
    assert r["tokens"] == greedy[:12]
    assert r["mat"] == [1] * 12                  # one token per call: the target's own


def test_bank_holding_the_greedy_continuation(tiny):
    case, root, greedy = tiny
    rng = np.random.default_rng(0)
    noise = [int(t) for t in rng.integers(2, case.cfg.vocab, size=60)]
    bank = noise + [EOS] + [root] + greedy + [EOS] + noise
    r = _run(case, root, 30, bank, depth=8, max_nodes=64)
    assert r["tokens"] == greedy[:30]
    # the root's occurrence before the greedy tokens proposes all 8 of them:
    # 8 accepted drafts plus the bonus on the first call
    assert r["mat"][0] == 9
    assert sum(r["mat"]) >= 30 and len(r["mat"]) < 30


@pytest.mark.parametrize("seed", range(3))
def test_lossless_under_misleading_hints(tiny, seed):
    """Banks of wrong continuations (the greedy trajectory with tokens
    replaced) and of noise: the committed output never changes."""
    case, root, greedy = tiny
    rng = np.random.default_rng(10 + seed)
    wrong = list(greedy)
    for i in rng.choice(len(wrong), size=6, replace=False):
        wrong[i] = int((wrong[i] + 1 + rng.integers(0, 50)) % case.cfg.vocab)
    bank = [root] + wrong + [EOS] + [int(t) for t in rng.integers(2, case.cfg.vocab, size=200)]
    native = [[int(t) for t in rng.integers(2, case.cfg.vocab, size=4)]]
    r = _run(case, root, 25, bank, native_lanes=native, depth=6, max_nodes=32)
    assert r["tokens"] == greedy[:25]
    assert all(m >= 1 for m in r["mat"])


def test_committed_cache_equals_plain_decoding(tiny):
    case, root, greedy = tiny
    bank = [root] + greedy + [EOS]
    r = _run(case, root, 20, bank, depth=5, max_nodes=32)
    n_new = len(r["cache_k"][0]) - case.ctx_len      # cached: the root and the committed tokens but the last
    steps, ck, cv = oracle.decode_sequence(case.view, case.cache_k64, case.cache_v64, case.ctx_len,
                                           [root] + greedy[:n_new - 1])
    for l in range(case.cfg.n_layers):
        np.testing.assert_allclose(r["cache_k"][l], ck[l], rtol=0, atol=1e-10)
        np.testing.assert_allclose(r["cache_v"][l], cv[l], rtol=0, atol=1e-10)
