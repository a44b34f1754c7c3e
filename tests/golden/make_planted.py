"""Write golden/planted.json: a root token and the target's own greedy
continuation per bf16 workload.

Calls only the CPU checker (oracle) on seeded synthetic inputs.  For each
workload (weights seed 0, synthetic committed cache) it draws candidate root
tokens from the seeded ROOT stream, k = 0, 1, ..., and decodes greedily from
each (Eq. 1 applied repeatedly) until `plant` tokens plus the bonus token are
found whose top-1/top-2 logit margins all exceed MIN_MARGIN.  A path with a
near-tie could be decided either way by a bf16 verifier, so exact comparison of
the accept outputs is only meaningful on such well-separated paths.

Usage: python tests/golden/make_planted.py [workload ...]
       python tests/golden/make_planted.py --roots N [--known i,j,...] workload ...

The second form writes golden/gated_roots.json instead: for each workload,
the first N roots of the seeded ROOT stream (weights seed 0, the workload's
own committed cache: a real prefill for the prefilled test models, the
synthetic cache otherwise) whose greedy continuation of `plant` tokens and
the bonus is well separated.  Every such root gives the GPU parity tests one
gated case: a tree around that path whose accept outputs must match exactly.
"""

import json
import os
import sys
import time

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
sys.path.insert(0, ROOT)
sys.path.insert(0, os.path.dirname(HERE))

import oracle  # noqa: E402
from cases import synthetic_cache, tiny_cache  # noqa: E402
from synth import gen  # noqa: E402
from synth.configs import WORKLOADS, workload  # noqa: E402
from synth.model import ROOT as ROOT_KIND, SynthModel  # noqa: E402

OUT = os.environ.get("PLANTED_OUT") or os.path.join(HERE, "planted.json")   # override: write elsewhere
ROOTS_OUT = os.environ.get("GATED_ROOTS_OUT") or os.path.join(HERE, "gated_roots.json")
MIN_MARGIN = 0.06       # the tests gate at 0.05
MAX_ROOTS = 64


def _separated_path(view, k64, v64, ctx_len, root, plant):
    """Greedy decisions after `root` until plant + 1 are found or one is a
    near-tie: (tokens, margins); complete when len(tokens) == plant + 1."""
    ck = [np.array(c) for c in k64]
    cv = [np.array(c) for c in v64]
    n_pos, tok, toks, margins = ctx_len, root, [], []
    while len(toks) < plant + 1:
        _, a, t1, t2, ks, vs = oracle.decode_step(view, ck, cv, n_pos, tok)
        margins.append(t1 - t2)
        if t1 - t2 <= MIN_MARGIN:
            break
        toks.append(a)
        ck = [np.concatenate([c, x[None]]) for c, x in zip(ck, ks)]
        cv = [np.concatenate([c, x[None]]) for c, x in zip(cv, vs)]
        n_pos += 1
        tok = a
    return toks, margins


def plant_one(name, seed=0):
    w = WORKLOADS[name]
    cfg = w.model
    view = SynthModel(cfg, seed).oracle_view()
    _, k64, v64 = synthetic_cache(cfg, seed, w.ctx_len)
    roots = gen.uniform_int(gen.tensor_key(seed, ROOT_KIND), MAX_ROOTS, cfg.vocab)
    for k in range(MAX_ROOTS):
        root = int(roots[k])
        toks, margins = _separated_path(view, k64, v64, w.ctx_len, root, w.plant)
        print("  %s root #%d: %d/%d decisions above margin" % (name, k, len(toks), w.plant + 1), flush=True)
        if len(toks) == w.plant + 1:
            return dict(seed=seed, ctx_len=w.ctx_len, root_index=k, root=root, planted=toks[:w.plant],
                        bonus=toks[w.plant], margins=margins,
                        note="oracle greedy continuation after the root on the synthetic cache; every margin "
                             "> %.2f" % MIN_MARGIN)
    raise RuntimeError("no well-separated greedy path found for %s" % name)


def gated_roots(name, n_cases, seed=0, max_roots=1024, known=(), on_found=None):
    """The first n_cases roots of the seeded ROOT stream whose greedy path
    (plant tokens and the bonus) is well separated.  `known`: root indices
    already found to qualify (checked again, and the search resumes after the
    last of them); on_found(result) is called after every qualifying root."""
    w = workload(name)
    cfg = w.model
    model = SynthModel(cfg, seed)
    view = model.oracle_view()
    if w.prefill:
        _, k64, v64 = tiny_cache(cfg, model, view, seed, w.ctx_len)
    else:
        _, k64, v64 = synthetic_cache(cfg, seed, w.ctx_len)
    roots = gen.uniform_int(gen.tensor_key(seed, ROOT_KIND), max_roots, cfg.vocab)
    found = []
    known = sorted(int(k) for k in known)
    order = known + list(range(known[-1] + 1 if known else 0, max_roots))

    def result():
        return dict(seed=seed, ctx_len=w.ctx_len, plant=w.plant, cases=list(found),
                    note="roots of the seeded stream whose oracle greedy continuation (plant tokens and "
                         "the bonus) has every top-1/top-2 margin > %.2f" % MIN_MARGIN)

    for k in order:
        root = int(roots[k])
        toks, margins = _separated_path(view, k64, v64, w.ctx_len, root, w.plant)
        if len(toks) == w.plant + 1:
            found.append(dict(root_index=k, root=root, planted=toks[:w.plant], bonus=toks[w.plant],
                              margins=margins))
            print("  %s root #%d kept (%d so far)" % (name, k, len(found)), flush=True)
            if on_found:
                on_found(result())
            if len(found) == n_cases:
                return result()
        elif k in known:
            raise RuntimeError("root #%d of %s no longer qualifies" % (k, name))
    raise RuntimeError("only %d well-separated roots for %s" % (len(found), name))


def main(names):
    data = {}
    if os.path.exists(OUT):
        with open(OUT) as f:
            data = json.load(f)
    for name in names:
        t0 = time.time()
        data[name] = plant_one(name)
        print(name, data[name]["planted"], ["%.3f" % m for m in data[name]["margins"]],
              "%.0fs" % (time.time() - t0), flush=True)
        with open(OUT, "w") as f:
            json.dump(data, f, indent=1)


def main_roots(n_cases, names, known=()):
    data = {}
    if os.path.exists(ROOTS_OUT):
        with open(ROOTS_OUT) as f:
            data = json.load(f)

    def save(name, r):
        data[name] = r
        with open(ROOTS_OUT, "w") as f:
            json.dump(data, f, indent=1)

    for name in names:
        t0 = time.time()
        save(name, gated_roots(name, n_cases, known=known, on_found=lambda r: save(name, r)))
        print(name, "%d roots" % n_cases, "%.0fs" % (time.time() - t0), flush=True)


if __name__ == "__main__":
    if len(sys.argv) > 2 and sys.argv[1] == "--roots":
        # --roots N [--known i,j,...] workload ...
        args = sys.argv[3:]
        known = ()
        if args and args[0] == "--known":
            known = [int(x) for x in args[1].split(",")]
            args = args[2:]
        main_roots(int(sys.argv[2]), args, known)
    else:
        main(sys.argv[1:] or [n for n, w in WORKLOADS.items() if w.model.dtype == "bf16"])
