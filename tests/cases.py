"""Seeded verify-step cases shared by the tests: model, cache, tree.

Inputs come from the seeded generator (synth); the planted greedy path and the
tiny model's prefilled cache come from the CPU checker (oracle) -- never from
the CUDA path.
"""

import dataclasses
import json
import os

import numpy as np

import oracle
from synth import gen, trees
from synth.configs import workload
from synth.model import PROMPT, ROOT, TREE_SHAPE, SynthModel, synthetic_kv

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


@dataclasses.dataclass
class Case:
    cfg: object
    model: SynthModel
    view: object                 # oracle view (fp64 tensors on request)
    ctx_len: int
    cache_native: list           # per layer (k, v) native arrays [ctx_len, nkv, d]
    cache_k64: list              # per layer fp64 arrays (same values)
    cache_v64: list
    tokens: np.ndarray
    parent: np.ndarray
    planted_path: list           # node ids root-first
    planted_margins: list


def round_cache(cfg, arr64):
    """Round a fp64 cache to the storage type; return (native, widened fp64)."""
    if cfg.kv_dtype == "f16":
        h = np.asarray(arr64, np.float32).astype(np.float16)
        return h.view(np.uint16), h.astype(np.float64)
    if cfg.dtype == "f32":
        a32 = np.asarray(arr64, np.float32)
        return a32, a32.astype(np.float64)
    bits = gen.np_f32_to_bf16_bits(np.asarray(arr64, np.float32))
    return bits, gen.bf16_bits_to_f64(bits)


def tiny_cache(cfg, model, view, seed, ctx_len):
    prompt = gen.uniform_int(gen.tensor_key(seed, PROMPT), ctx_len, cfg.vocab)
    ck, cv, _ = oracle.prefill(view, prompt)
    native, k64, v64 = [], [], []
    for l in range(cfg.n_layers):
        kn, kw = round_cache(cfg, ck[l])
        vn, vw = round_cache(cfg, cv[l])
        native.append((kn, vn))
        k64.append(kw)
        v64.append(vw)
    return native, k64, v64


def synthetic_cache(cfg, seed, ctx_len):
    native, k64, v64 = [], [], []
    for l in range(cfg.n_layers):
        native.append((synthetic_kv(cfg, seed, l, ctx_len, "native", "k"),
                       synthetic_kv(cfg, seed, l, ctx_len, "native", "v")))
        k64.append(synthetic_kv(cfg, seed, l, ctx_len, "f64", "k"))
        v64.append(synthetic_kv(cfg, seed, l, ctx_len, "f64", "v"))
    return native, k64, v64


def root_token(cfg, seed):
    return int(gen.uniform_int(gen.tensor_key(seed, ROOT), 1, cfg.vocab)[0])


def build_case(name="tiny", seed=0, T=None, recipe=None, plant=None, ctx_len=None,
               cfg_overrides=None, gain_std=0.0, planted=None, prefill=None, root=None, tree_key=None):
    """A verify-step case for workload `name` (defaults from its recipe)."""
    w = workload(name)
    cfg = w.model if not cfg_overrides else dataclasses.replace(w.model, **cfg_overrides)
    T = w.T if T is None else T
    recipe = w.tree if recipe is None else recipe
    plant = w.plant if plant is None else plant
    ctx_len = w.ctx_len if ctx_len is None else ctx_len
    prefill = w.prefill if prefill is None else prefill
    model = SynthModel(cfg, seed, gain_std=gain_std)
    view = model.oracle_view()
    if prefill:
        native, k64, v64 = tiny_cache(cfg, model, view, seed, ctx_len)
    else:
        native, k64, v64 = synthetic_cache(cfg, seed, ctx_len)
    root = root_token(cfg, seed) if root is None else int(root)
    if planted is None:
        if plant > 0:
            planted, margins = oracle.greedy_continuation(view, k64, v64, ctx_len, root, plant)
        else:
            planted, margins = [], []
    else:
        planted, margins = planted
    if tree_key is None:
        tree_key = gen.tensor_key(seed, TREE_SHAPE, T)
    tokens, parent, path = trees.make_tree(recipe, T, root, planted, cfg.vocab, tree_key)
    return Case(cfg, model, view, ctx_len, native, k64, v64, tokens, parent, path,
                list(margins))


def with_tree(case, name, root, planted, margins, index):
    """The same model and cache with another tree: the workload's recipe
    around root -> planted path, shape drawn from stream `index`."""
    w = workload(name)
    T = len(case.tokens)
    tokens, parent, path = trees.make_tree(w.tree, T, int(root), list(planted), case.cfg.vocab,
                                           gen.tensor_key(1000 + int(index), TREE_SHAPE, T))
    return dataclasses.replace(case, tokens=tokens, parent=parent, planted_path=path,
                               planted_margins=list(margins))


def load_planted(name):
    """Planted greedy paths written by golden/make_planted.py (oracle only)."""
    with open(os.path.join(GOLDEN, "planted.json")) as f:
        d = json.load(f)
    return d[name]


def load_gated_roots(name):
    """Well-separated roots and their greedy paths, written by
    golden/make_planted.py --roots (oracle only)."""
    with open(os.path.join(GOLDEN, "gated_roots.json")) as f:
        d = json.load(f)
    return d[name]
