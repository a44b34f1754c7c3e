"""Hint-bank candidate step on the GPU (oos_hint_tree) against the oracle:
the packed tree, its size and the match/lane counts, bit for bit."""

import os
import sys

import numpy as np
import pytest

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))

from oracle import hint_bank as hb  # noqa: E402

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
from paper_2608_00814_gb300 import binding as B  # noqa: E402


def _gpu(bank, eos, y, native, max_lanes, depth, max_nodes):
    dev = "cuda"
    b = torch.as_tensor(np.asarray(bank, np.int32), device=dev)
    p = torch.as_tensor(np.asarray(y, np.int32), device=dev)
    if native:
        stride = max(1, max(len(l) for l in native))
        nat = np.full((len(native), stride), -7, np.int32)
        for i, l in enumerate(native):
            nat[i, :len(l)] = l
        nat_t = torch.as_tensor(nat, device=dev)
        nl_t = torch.as_tensor(np.array([len(l) for l in native], np.int32), device=dev)
    else:
        nat_t = nl_t = None
    ws = torch.empty(B.oos_hint_workspace_bytes(len(bank)), dtype=torch.uint8, device=dev)
    tok = torch.full((max_nodes,), -5, dtype=torch.int32, device=dev)
    par = torch.full((max_nodes,), -5, dtype=torch.int32, device=dev)
    T = torch.zeros(1, dtype=torch.int32, device=dev)
    info = torch.zeros(3, dtype=torch.int32, device=dev)
    B.oos_hint_tree(b, eos, p, nat_t, nl_t, max_lanes, depth, max_nodes, ws, tok, par, T, info)
    torch.cuda.synchronize()
    n = int(T.item())
    return tok[:n].cpu().numpy(), par[:n].cpu().numpy(), info.cpu().numpy().tolist(), tok[n:].cpu().numpy()


def _check(bank, eos, y, native, max_lanes, depth, max_nodes):
    r = hb.propose_tree(bank, eos, y, native, max_lanes, depth, max_nodes)
    tok, par, info, rest = _gpu(bank, eos, y, native, max_lanes, depth, max_nodes)
    np.testing.assert_array_equal(tok, r["tokens"])
    np.testing.assert_array_equal(par, r["parents"])
    assert info == [r["match_n"], r["hint_lanes"], r["lanes"]]
    assert np.all(rest == -5)          # nothing written past T
    return r


def test_hand_fixtures():
    bank = [5, 6, 7, 8, 0, 9, 6, 7, 10, 11, 0, 6, 7]
    r = _check(bank, 0, [4, 6, 7], [[8, 2], [30]], 3, 4, 64)
    assert r["tokens"].tolist() == [7, 8, 10, 11, 2]
    _check(bank, 0, [1, 2, 9, 6, 7], [], 8, 8, 128)
    _check([1, 2, 3, 4, 0, 1, 2, 3, 4], 0, [1], [], 8, 3, 3)
    _check([1, 2, 0], 0, [9], [[4, 5], [4, 6]], 8, 4, 8)


@pytest.mark.parametrize("seed", range(8))
def test_random_banks(seed):
    rng = np.random.default_rng(seed)
    vocab = int(rng.integers(3, 12))
    bank = rng.integers(0, vocab, size=int(rng.integers(1, 3000))).tolist()   # many 256-position rounds
    y = rng.integers(0, vocab, size=int(rng.integers(1, 12))).tolist()
    native = [rng.integers(1, vocab, size=int(rng.integers(0, 9))).tolist() for _ in range(int(rng.integers(0, 5)))]
    _check(bank, 0, y, native, int(rng.integers(0, 12)), int(rng.integers(1, 20)), int(rng.integers(1, 129)))


def test_large_bank_with_planted_views():
    """A 50k-token bank of 400 views over a 32k vocabulary; the prefix's last
    7 tokens occur in three views, with different continuations."""
    rng = np.random.default_rng(42)
    vocab, eos = 32000, 2
    views = [rng.integers(3, vocab, size=int(rng.integers(60, 190))).tolist() for _ in range(400)]
    key = rng.integers(3, vocab, size=7).tolist()
    for v, cont in ((17, [101, 102, 103]), (233, [101, 104]), (390, [555, 556, 557, 558])):
        views[v][20:20 + 7 + len(cont)] = key + cont
    bank = []
    for v in views:
        bank += v + [eos]
    y = rng.integers(3, vocab, size=30).tolist() + key
    r = _check(bank, eos, y, [[7, 8, 9]], 8, 12, 128)
    assert r["match_n"] == 7 and r["hint_lanes"] == 3


def test_edges():
    _check([4], 0, [4], [], 4, 4, 8)                        # one-token bank: nothing follows
    _check([4, 5, 6], 0, [4, 5], [[1]], 4, 4, 1)            # root only
    _check([4, 5, 6], 0, [4, 5], [[1]], 0, 4, 8)            # no lanes allowed
    _check([3, 3, 3, 3, 3], 0, [3] * 9, [], 4, 4, 16)       # overlapping occurrences, suffix capped at 7


@pytest.mark.parametrize("spots", [(3_000, 140_000, 290_000), (299_000,)])
def test_bank_over_several_spans(spots):
    """A 300k-token bank covers five 65536-position spans of the kernel's
    summaries; occurrences in the first, middle and last (partial) spans, or
    in the last one only."""
    rng = np.random.default_rng(len(spots))
    vocab, eos = 50000, 1
    bank = rng.integers(2, vocab, size=300_000)
    key = rng.integers(2, vocab, size=7)
    for i, at in enumerate(spots):
        bank[at:at + 7] = key
        bank[at + 7:at + 10] = [40 + i, 41, 42]
    y = np.concatenate([rng.integers(2, vocab, size=12), key]).tolist()
    r = _check(bank.tolist(), eos, y, [[5, 6]], 6, 8, 96)
    assert r["match_n"] == 7 and r["hint_lanes"] == len(spots)
