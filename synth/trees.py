"""Seeded candidate-tree generators (topologically numbered, root = node 0).

A tree is (tokens[T], parent[T]) with parent[0] = -1 and parent[i] < i.  The
paper packs schema, retrieved and hint continuations into one tree but gives
no packing order; these generators stand in for that traffic with the shapes
of the benchmark workloads.  Each tree holds one planted path below the root
whose tokens the caller supplies (the model's own greedy continuation, so the
verifier should accept it); all other draft tokens are uniform-random and
siblings never share a token.  A final random topological renumbering makes
accepted node ids differ from their depths, which exercises KV compaction.

Randomness comes from the SplitMix64 stream of gen.py, so trees are identical
on every host.
"""

import numpy as np

from . import gen


class Rng:
    def __init__(self, key):
        self.key = key & gen.M64
        self.i = 0

    def next64(self):
        r = gen.stream_at(self.key, self.i)
        self.i += 1
        return r

    def randint(self, lo, hi):
        """Uniform integer in [lo, hi] (inclusive)."""
        n = hi - lo + 1
        return lo + (((self.next64() >> 32) * n) >> 32)

    def choice(self, seq):
        return seq[self.randint(0, len(seq) - 1)]


def _relabel(parent_of, root_first_order_rng, planted_nodes, tries=64):
    """Random topological renumbering; returns old->new map."""
    n = len(parent_of)
    children = [[] for _ in range(n)]
    for v in range(1, n):
        children[parent_of[v]].append(v)
    best = None
    for _ in range(tries):
        avail = [0]
        order = []
        while avail:
            k = root_first_order_rng.randint(0, len(avail) - 1)
            v = avail.pop(k)
            order.append(v)
            avail.extend(children[v])
        new = [0] * n
        for i, v in enumerate(order):
            new[v] = i
        best = new
        # want at least one accepted-path node whose id differs from its depth
        if any(new[v] != j for j, v in enumerate(planted_nodes)) or len(planted_nodes) == n:
            break
    return best


def _finish(parent_of, tok_of, planted_nodes, rng):
    new = _relabel(parent_of, rng, planted_nodes)
    n = len(parent_of)
    tokens = np.zeros(n, np.int32)
    parent = np.zeros(n, np.int32)
    for v in range(n):
        tokens[new[v]] = tok_of[v]
        parent[new[v]] = -1 if v == 0 else new[parent_of[v]]
    path = [new[v] for v in planted_nodes]
    return tokens, parent, path


def _draw_token(rng, vocab, taken):
    while True:
        t = rng.randint(0, vocab - 1)
        if t not in taken:
            return t


def make_tree(recipe, T, root_token, planted, vocab, key):
    """Build one tree.

    recipe: dict(kind="uniform", max_depth) | dict(kind="branch", bmin, bmax,
            max_depth) | dict(kind="wide", level_branch, max_depth) | dict(kind="chain").
    planted: tokens of the planted path below the root (depth 1..len).
    Returns (tokens int32[T], parent int32[T], planted_path node ids incl. root).
    """
    rng = Rng(key)
    planted = [int(t) for t in planted]
    kind = recipe["kind"]
    max_depth = recipe.get("max_depth", T)
    if len(planted) > min(T - 1, max_depth):
        raise ValueError("planted path does not fit the tree")
    parent_of = [-1]
    depth = [0]
    tok_of = [int(root_token)]
    kids = [[]]

    def add(p, tok):
        parent_of.append(p)
        depth.append(depth[p] + 1)
        tok_of.append(tok)
        kids.append([])
        kids[p].append(len(parent_of) - 1)
        return len(parent_of) - 1

    def add_random(p):
        taken = {tok_of[c] for c in kids[p]}
        return add(p, _draw_token(rng, vocab, taken))

    # planted chain first
    chain = [0]
    for t in planted:
        chain.append(add(chain[-1], t))
    leaf = chain[-1] if planted else None

    if kind == "chain":
        while len(parent_of) < T:
            tail = len(parent_of) - 1
            add_random(tail)
    elif kind == "uniform":
        while len(parent_of) < T:
            cands = [v for v in range(len(parent_of)) if depth[v] < max_depth and v != leaf]
            add_random(rng.choice(cands))
    elif kind == "branch":
        bmin, bmax = recipe["bmin"], recipe["bmax"]
        while len(parent_of) < T:
            queue = [0]
            grew = False
            while queue and len(parent_of) < T:
                v = queue.pop(0)
                if depth[v] < max_depth and v != leaf:
                    want = rng.randint(bmin, bmax)
                    while len(kids[v]) < want and len(parent_of) < T:
                        add_random(v)
                        grew = True
                queue.extend(kids[v])
            if not grew:
                raise ValueError("tree recipe cannot reach T nodes")
    elif kind == "wide":
        b = recipe["level_branch"]
        # level 1 and level 2, full (planted chain already holds one node of each)
        for v in [0]:
            while len(kids[v]) < b and len(parent_of) < T:
                add_random(v)
        for v in list(kids[0]):
            while len(kids[v]) < b and len(parent_of) < T and v != leaf:
                add_random(v)
        level2 = [v for v in range(len(parent_of)) if depth[v] == 2 and v != leaf]
        # remaining nodes: chains hanging under random level-2 nodes
        while len(parent_of) < T:
            v = rng.choice(level2)
            while kids[v] and len(parent_of) < T:
                v = rng.choice(kids[v])
                if v == leaf or depth[v] >= max_depth:
                    break
            if v == leaf or depth[v] >= max_depth:
                continue
            length = rng.randint(1, max_depth - depth[v])
            for _ in range(length):
                if len(parent_of) >= T:
                    break
                v = add_random(v)
    else:
        raise ValueError(kind)
    return _finish(parent_of, tok_of, chain, rng)


def random_tokens_tree(T, vocab, key, max_depth=None):
    """A tree with parents uniform over earlier nodes and all tokens random."""
    rng = Rng(key)
    parent = np.full(T, -1, np.int32)
    depth = [0]
    tokens = np.zeros(T, np.int32)
    tokens[0] = rng.randint(0, vocab - 1)
    kids = {0: set()}
    for i in range(1, T):
        cands = [v for v in range(i) if max_depth is None or depth[v] < max_depth]
        p = rng.choice(cands)
        parent[i] = p
        depth.append(depth[p] + 1)
        t = _draw_token(rng, vocab, kids[p])
        kids[p].add(t)
        kids[i] = set()
        tokens[i] = t
    return tokens, parent
