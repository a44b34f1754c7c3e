"""CPU checker for the multi-step decode loop -- TEST INFRASTRUCTURE ONLY.

Only the test suite, `__graft_entry__.smoke()` and the benchmark's CPU legs
may import it; the product path never does.

The loop (Section 2, "The ToolSpec decoding loop"; Section 4, "Verify and
commit"): at every candidate-construction boundary a tree is built from
everything committed so far -- here from the hint bank (oracle/hint_bank.py)
and optional native lanes -- the target verifies it in one pass, the longest
greedy-approved prefix is committed with the target's own next token (the
bonus), and only the accepted path's K/V enter the cache.  The bonus is the
next round's root.  #MAT (Section 5, "Metrics and Correctness Audit") is the
number of tokens a verification call commits: the accepted path (root
included) -- its draft nodes plus the bonus.

Readings (also in the design notes): the root's K/V is written by the call
that verifies it (it was committed as the previous call's bonus, or is the
prompt's last token); a round's committed tokens are the accepted path's
draft tokens followed by the bonus; the loop stops once n_tokens tokens are
committed and returns exactly n_tokens of them.
"""

import numpy as np

from .hint_bank import propose_tree
from .tree_verify import verify_and_accept


def speculative_decode(m, cache_k, cache_v, n_pos, root, n_tokens, bank, eos, native_lanes=(), max_lanes=8,
                       depth=16, max_nodes=64):
    """Commit n_tokens tokens after `root` with tree verification.

    cache_k / cache_v: per layer [>= n_pos, nkv, d], positions [0, n_pos)
    committed; root: the last committed token (not cached yet).  The bank is
    matched against the committed tokens known here: the root and what the
    loop commits (the prompt before it is not re-read).  Returns a dict with
    tokens (the n_tokens committed tokens), mat (tokens committed by each
    verification call), cache_k / cache_v (committed positions only).
    """
    ck = [np.array(c[:n_pos]) for c in cache_k]
    cv = [np.array(c[:n_pos]) for c in cache_v]
    committed = [int(root)]           # root first; the tree's root is always the last entry
    out, mat = [], []
    while len(out) < n_tokens:
        tree = propose_tree(bank, eos, committed, list(native_lanes), max_lanes, depth, max_nodes)
        tokens, parents = tree["tokens"], tree["parents"]
        r = verify_and_accept(m, ck, cv, n_pos, tokens, parents)
        L = int(r["accepted_len"])
        nodes = [int(i) for i in r["accepted_nodes"][:L]]
        # the accepted path's K/V (root included) enter the cache, nothing else does
        ck = [np.concatenate([c, tk[nodes]]) for c, tk in zip(ck, r["tree_k"])]
        cv = [np.concatenate([c, tv[nodes]]) for c, tv in zip(cv, r["tree_v"])]
        n_pos += L
        new = [int(t) for t in r["accepted_tokens"][1:L]] + [int(r["bonus"])]
        committed += new
        out += new
        mat.append(L)
    return dict(tokens=out[:n_tokens], mat=mat, cache_k=ck, cache_v=cv)
