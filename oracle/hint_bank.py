"""CPU checker for the hint-bank candidate step -- TEST INFRASTRUCTURE ONLY.

Only the test suite, `__graft_entry__.smoke()` and the benchmark's CPU legs
may import it; the product path never does.

What it computes (the paper's "Suffix matching" and "Candidate boundary"
paragraphs, Section 4): the target's committed prefix y is matched against a
request-level hint bank -- the tokenised views joined by the target's EOS
token -- and the tokens that follow a match become candidate continuations
("lanes") of the next verification tree, ahead of the verifier's native
candidates, under a fixed lane budget B (Merge_B).

Readings where the paper is silent (each one also listed in the design notes):
  * An occurrence of suffix_n(y) ends at bank index p and counts only when a
    continuation follows it: p + 1 < len(bank) and bank[p + 1] != EOS.
  * n runs from 7 down to 1 (never above len(y)); the first n with at least
    one counted occurrence is used, and only its occurrences propose lanes.
  * Occurrences are taken in bank order.  A lane is bank[p+1 : p+1+D] cut
    before the first EOS (D = the lane depth).
  * Lanes are merged into a prefix tree rooted at the last committed token
    y[-1]; a node is numbered when it is created (root 0), so parents come
    before children.  A lane counts towards B only when it creates a node; a
    lane that repeats (a prefix of) an earlier one is skipped.  Native lanes
    follow the hint lanes under the same rules until B lanes or the node
    budget are reached; a lane cut by the node budget keeps its first nodes.
"""

import numpy as np


def suffix_match(bank, eos, y, n_max=7):
    """(n, positions): the longest n <= min(n_max, len(y)) whose length-n
    suffix of y occurs in the bank with a continuation after it, and the bank
    indices p (ascending) where those occurrences end.  (0, []) when no n has
    one.  Brute force: every position, every n."""
    bank = [int(t) for t in bank]
    y = [int(t) for t in y]
    for n in range(min(n_max, len(y)), 0, -1):
        s = y[-n:]
        pos = []
        for p in range(n - 1, len(bank)):
            if bank[p - n + 1:p + 1] == s and p + 1 < len(bank) and bank[p + 1] != eos:
                pos.append(p)
        if pos:
            return n, pos
    return 0, []


def continuation(bank, eos, p, depth):
    """Tokens after bank index p: at most `depth`, stopping before an EOS."""
    out = []
    for q in range(p + 1, min(len(bank), p + 1 + depth)):
        if int(bank[q]) == eos:
            break
        out.append(int(bank[q]))
    return out


def pack_tree(root, lanes, max_lanes, max_nodes):
    """Prefix-tree packing of candidate lanes (token lists continuing `root`).

    Returns (tokens, parents, n_lanes_used, lane_used[i]): node 0 is the root
    (parent -1); each new node's parent was created before it."""
    tokens, parents = [int(root)], [-1]
    children = {}            # (parent node, token) -> node
    used = 0
    lane_used = []
    for lane in lanes:
        if used >= max_lanes or len(tokens) >= max_nodes:
            lane_used.append(False)
            continue
        cur, created = 0, False
        for t in lane:
            key = (cur, int(t))
            if key in children:
                cur = children[key]
                continue
            if len(tokens) >= max_nodes:
                break
            tokens.append(int(t))
            parents.append(cur)
            children[key] = len(tokens) - 1
            cur = len(tokens) - 1
            created = True
        lane_used.append(created)
        used += int(created)
    return tokens, parents, used, lane_used


def propose_tree(bank, eos, y, native_lanes, max_lanes, depth, max_nodes, n_max=7):
    """The next verification tree: hint lanes from the longest aligned suffix
    match first, native lanes after them (Merge_B).  Returns a dict with
    tokens, parents, match_n, hint_lanes (hint lanes that created a node)."""
    n, pos = suffix_match(bank, eos, y, n_max)
    hint = [continuation(bank, eos, p, depth) for p in pos]
    lanes = hint + [list(map(int, l))[:depth] for l in native_lanes]
    tokens, parents, used, lane_used = pack_tree(int(y[-1]), lanes, max_lanes, max_nodes)
    return dict(tokens=np.array(tokens, np.int32), parents=np.array(parents, np.int32), match_n=n,
                hint_lanes=int(sum(lane_used[:len(hint)])), lanes=used)
