"""Pins of the hint-bank candidate checker (oracle/hint_bank.py) -- no GPU.

Hand-worked fixtures, an independent string-search restatement of the
suffix match, and structural invariants of the packed tree."""

import os
import sys

import numpy as np
import pytest

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))

from oracle import hint_bank as hb  # noqa: E402

EOS = 0


def test_hand_fixture_longest_aligned_suffix():
    # bank: views [5 6 7 8] [9 6 7 10 11] [6 7] joined by EOS (0)
    bank = [5, 6, 7, 8, 0, 9, 6, 7, 10, 11, 0, 6, 7]
    # y ends with 9 6 7: suffix 3 "9 6 7" ends at index 7, followed by 10
    n, pos = hb.suffix_match(bank, EOS, [1, 2, 9, 6, 7])
    assert (n, pos) == (3, [7])
    # y ends with 4 6 7: "4 6 7" never occurs; "6 7" ends at 2 (-> 8), 7 (-> 10) and
    # 12 (bank end: no continuation, not counted)
    n, pos = hb.suffix_match(bank, EOS, [4, 6, 7])
    assert (n, pos) == (2, [2, 7])
    # a suffix only ever followed by EOS counts as no match at that length: "3 4"
    # ends at 1 before an EOS; "4" ends at 1 (EOS next) and at 3 (5 next)
    n, pos = hb.suffix_match([3, 4, 0, 4, 5], EOS, [3, 4])
    assert (n, pos) == (1, [3])


def test_hand_fixture_tree():
    bank = [5, 6, 7, 8, 0, 9, 6, 7, 10, 11, 0, 6, 7]
    r = hb.propose_tree(bank, EOS, [4, 6, 7], native_lanes=[[8, 2], [30]], max_lanes=3, depth=4,
                        max_nodes=64)
    # hint lanes: after index 2 -> [8] (stops at EOS); after index 7 -> [10, 11]
    # native lanes: [8, 2] shares 8 with the first lane, [30] would be a 4th lane
    assert r["match_n"] == 2 and r["hint_lanes"] == 2 and r["lanes"] == 3
    assert r["tokens"].tolist() == [7, 8, 10, 11, 2]
    assert r["parents"].tolist() == [-1, 0, 0, 2, 1]


def test_hand_fixture_budgets():
    # node budget cuts a lane after its first nodes; duplicate lanes do not count
    r = hb.propose_tree([1, 2, 3, 4, 0, 1, 2, 3, 4], EOS, [1], native_lanes=[], max_lanes=8, depth=3,
                        max_nodes=3)
    # "1" ends at 0 and 5; both continue 2 3 4 -> one lane, cut to 2 new nodes
    assert r["match_n"] == 1 and r["tokens"].tolist() == [1, 2, 3] and r["parents"].tolist() == [-1, 0, 1]
    assert r["hint_lanes"] == 1
    # no aligned match at all: native lanes only
    r = hb.propose_tree([1, 2, 0], EOS, [9], native_lanes=[[4, 5], [4, 6]], max_lanes=8, depth=4, max_nodes=8)
    assert r["match_n"] == 0 and r["hint_lanes"] == 0
    assert r["tokens"].tolist() == [9, 4, 5, 6] and r["parents"].tolist() == [-1, 0, 1, 1]


def _find_all(hay, needle):
    """End indices of every occurrence, by str.find on a fixed-width encoding."""
    enc = lambda xs: "".join("%06d," % x for x in xs)
    h, nd = enc(hay), enc(needle)
    out, i = [], h.find(nd)
    while i >= 0:
        if i % 7 == 0:
            out.append(i // 7 + len(needle) - 1)
        i = h.find(nd, i + 1)
    return out


@pytest.mark.parametrize("seed", range(6))
def test_suffix_match_against_string_search(seed):
    rng = np.random.default_rng(seed)
    vocab = 6 + seed                       # small vocabularies: many partial matches
    bank = rng.integers(0, vocab, size=400).tolist()
    y = rng.integers(1, vocab, size=9).tolist()
    n, pos = hb.suffix_match(bank, EOS, y)
    want_n, want_pos = 0, []
    for m in range(7, 0, -1):
        ends = [p for p in _find_all(bank, y[-m:]) if p + 1 < len(bank) and bank[p + 1] != EOS]
        if ends:
            want_n, want_pos = m, ends
            break
    assert (n, pos) == (want_n, want_pos)


@pytest.mark.parametrize("seed", range(6))
def test_packed_tree_is_the_trie_of_its_lanes(seed):
    rng = np.random.default_rng(100 + seed)
    bank = rng.integers(0, 5, size=300).tolist()
    y = rng.integers(1, 5, size=6).tolist()
    native = [rng.integers(1, 5, size=int(rng.integers(1, 6))).tolist() for _ in range(4)]
    r = hb.propose_tree(bank, EOS, y, native, max_lanes=6, depth=5, max_nodes=40)
    tok, par = r["tokens"].tolist(), r["parents"].tolist()
    assert par[0] == -1 and tok[0] == y[-1]
    assert all(0 <= par[i] < i for i in range(1, len(tok)))
    # every node's root path (without the root) is a prefix of some lane, and siblings differ
    n, pos = hb.suffix_match(bank, EOS, y)
    lanes = [tuple(hb.continuation(bank, EOS, p, 5)) for p in pos] + [tuple(l[:5]) for l in native]
    paths = {}
    for i in range(1, len(tok)):
        paths[i] = paths.get(par[i], ()) + (tok[i],)
        assert any(l[:len(paths[i])] == paths[i] for l in lanes)
    assert len(set(paths.values())) == len(paths)
    assert len(tok) <= 40 and r["lanes"] <= 6
