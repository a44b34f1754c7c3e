"""CUDA path vs the CPU checker, element by element, through the C ABI."""

import json
import os

import numpy as np
import pytest
import torch

import oracle
from cases import GOLDEN, build_case, load_gated_roots, load_planted, with_tree
from gpu_util import (GATE, TOL, check_case, check_compaction, gpu_cache, gpu_model, max_rel_err, ok_nodes, run,
                      to_f64)
from synth import trees

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a GPU", allow_module_level=True)

from paper_2608_00814_gb300 import binding as B  # noqa: E402


def _oracle(case, only=None):
    return oracle.verify_tree(case.view, case.cache_k64, case.cache_v64, case.ctx_len, case.tokens, case.parent,
                              only=only)


# ------------------------------------------------------------------ tiny fp32 decoder

@pytest.fixture(scope="module")
def tiny_models():
    """One GPU model per weight seed/variant, reused across tests."""
    return {}


def _tiny(tiny_models, seed, **kw):
    case = build_case("tiny", seed, **kw)
    key = (seed, tuple(sorted((kw.get("cfg_overrides") or {}).items())), kw.get("gain_std", 0.0))
    if key not in tiny_models:
        tiny_models[key] = gpu_model(case)
    return case, tiny_models[key][0]


def test_tiny_parity_many_seeds(tiny_models):
    gated = 0
    for seed in range(24):
        case, model = _tiny(tiny_models, seed)
        kv = gpu_cache(case, case.ctx_len + 128)
        g = run(model, kv, case.ctx_len, case.tokens, case.parent)
        r = _oracle(case)
        gated += check_case(case, g, r)
        check_compaction(model, kv, case.ctx_len, g)
    assert gated >= 20


@pytest.mark.parametrize("overrides,gain_std", [(dict(qk_norm=True), 0.0), (dict(qkv_bias=True), 0.2),
                                                (dict(qk_norm=True, qkv_bias=True, tied=True), 0.2),
                                                # Llama-3.1 rotary rescaling, short original context so
                                                # that all three frequency regions occur
                                                (dict(rope_factor=8.0, rope_orig_max_pos=64), 0.0)])
def test_tiny_variants(tiny_models, overrides, gain_std):
    case, model = _tiny(tiny_models, 3, cfg_overrides=overrides, gain_std=gain_std)
    kv = gpu_cache(case, case.ctx_len + 128)
    g = run(model, kv, case.ctx_len, case.tokens, case.parent)
    check_case(case, g, _oracle(case))
    check_compaction(model, kv, case.ctx_len, g)


@pytest.mark.parametrize("T,recipe,ctx", [
    (1, dict(kind="chain"), 128),                       # vanilla decode step
    (13, dict(kind="uniform", max_depth=5), 128),        # ragged tree
    (37, dict(kind="branch", bmin=1, bmax=4, max_depth=9), 128),
    (100, dict(kind="uniform", max_depth=30), 128),
    (128, dict(kind="branch", bmin=1, bmax=3, max_depth=40), 128),   # largest tree
    (128, dict(kind="chain"), 128),                     # deepest tree: depth 127
    (64, dict(kind="wide", level_branch=8, max_depth=16), 128),
    (9, dict(kind="uniform", max_depth=4), 0),           # empty cache
    (20, dict(kind="uniform", max_depth=6), 1),          # one cached position
    (16, dict(kind="uniform", max_depth=6), 333),        # cache not a multiple of any tile
])
def test_tiny_shapes(tiny_models, T, recipe, ctx):
    case, model = _tiny(tiny_models, 1, T=T, recipe=recipe, ctx_len=ctx, plant=min(3, T - 1))
    kv = gpu_cache(case, ctx + T + 5)
    g = run(model, kv, ctx, case.tokens, case.parent)
    check_case(case, g, _oracle(case))
    check_compaction(model, kv, ctx, g)


def test_tiny_star_and_duplicate_siblings(tiny_models):
    case, model = _tiny(tiny_models, 2, T=8)
    r = _oracle(case)
    # star: every draft a child of the root, two of them carrying the greedy token
    tokens = np.array([case.tokens[0]] + [(int(r["argmax"][0]) + k) % case.cfg.vocab for k in range(7)], np.int32)
    tokens[3] = r["argmax"][0]
    parent = np.array([-1] + [0] * 7, np.int32)
    case.tokens, case.parent = tokens, parent
    kv = gpu_cache(case, case.ctx_len + 8)
    g = run(model, kv, case.ctx_len, tokens, parent)
    rr = _oracle(case)
    check_case(case, g, rr)
    if rr["top1"][0] - rr["top2"][0] > GATE["f32"]:
        assert g["accepted_nodes"][:2] == [0, 1]      # lowest id among equally deep accepted nodes


def test_tiny_invalid_trees(tiny_models):
    case, model = _tiny(tiny_models, 0)
    kv = gpu_cache(case, case.ctx_len + 8)
    bad = [
        (case.tokens, np.array([0, 0, 0, 1, 1, 2, 2, 3], np.int32)),            # root has a parent
        (case.tokens, np.array([-1, 0, 0, 5, 1, 2, 2, 3], np.int32)),           # parent after child
        (case.tokens, np.array([-1, 0, 0, 3, 1, 2, 2, 3], np.int32)),           # self parent
        (np.array([1, 2, 3, case.cfg.vocab, 5, 6, 7, 8], np.int32), case.parent),  # token out of range
        (np.array([1, -2, 3, 4, 5, 6, 7, 8], np.int32), case.parent),
    ]
    for tokens, parent in bad:
        g = run(model, kv, case.ctx_len, tokens, parent)
        assert g["status"] == B.OOS_ETREE
        assert g["accepted_len"] == 0 and g["bonus"] == -1
        assert all(x == -1 for x in g["accepted_nodes"])
    # the handle stays usable after a rejected tree
    g = run(model, kv, case.ctx_len, case.tokens, case.parent)
    assert g["status"] == B.OOS_OK and g["accepted_len"] >= 1


def test_host_side_errors(tiny_models):
    case, model = _tiny(tiny_models, 0)
    kv = gpu_cache(case, case.ctx_len + 8)
    tok = torch.as_tensor(case.tokens, device="cuda")
    par = torch.as_tensor(case.parent, device="cuda")
    outs = B.VerifyOutputs(8)
    with pytest.raises(B.OosError) as e:
        B.oos_tree_verify(model, kv, case.ctx_len + 1, tok, par, 8, outs.accepted_len, outs.accepted_nodes,
                          outs.accepted_tokens, outs.bonus)
    assert e.value.code == B.OOS_ECAPACITY
    for T, ctx in ((0, 10), (129, 0), (8, -1)):
        with pytest.raises(B.OosError) as e:
            B.oos_tree_verify(model, kv, ctx, tok, par, T, outs.accepted_len, outs.accepted_nodes,
                              outs.accepted_tokens, outs.bonus)
        assert e.value.code == B.OOS_EINVAL
    with pytest.raises(B.OosError) as e:
        B.oos_tree_verify(model, kv, 0, None, par, 8, outs.accepted_len, outs.accepted_nodes, outs.accepted_tokens,
                          outs.bonus)
    assert e.value.code == B.OOS_EINVAL


def test_graph_replay_matches_direct_launch(tiny_models):
    case, model = _tiny(tiny_models, 5)
    direct = B.OosModel(case.cfg, tiny_models[(5, (), 0.0)][1], use_graph=False)
    kv1 = gpu_cache(case, case.ctx_len + 8)
    kv2 = gpu_cache(case, case.ctx_len + 8)
    a = run(model, kv1, case.ctx_len, case.tokens, case.parent)
    a2 = run(model, kv1, case.ctx_len, case.tokens, case.parent)   # replay of the captured graph
    b = run(direct, kv2, case.ctx_len, case.tokens, case.parent)
    for x in (a2, b):
        assert np.array_equal(a["final_hidden"], x["final_hidden"])
        assert np.array_equal(a["argmax"], x["argmax"])
        assert a["accepted_nodes"] == x["accepted_nodes"] and a["bonus"] == x["bonus"]



@pytest.mark.parametrize("name,overrides", [("tiny", None), ("mini-bf16", None),
                                            ("mini-bf16", dict(cache_dtype="f16"))])
def test_graph_reused_across_committed_lengths(name, overrides):
    """oos_tree_verify keeps its captured graph when only the committed length
    changes (the new length goes to the tree-prep node alone) and captures
    again when the length changes the attention's split count.  Every call,
    with the same output buffers, equals a direct launch bit for bit and the
    checker at its own length."""
    case = build_case(name, 0, cfg_overrides=overrides)
    graph_model, w = gpu_model(case)
    direct = B.OosModel(case.cfg, w, use_graph=False)
    T = len(case.tokens)
    kv_g = gpu_cache(case, case.ctx_len + T)
    kv_d = gpu_cache(case, case.ctx_len + T)
    snap = [t.clone() for t in kv_g.k], [t.clone() for t in kv_g.v]
    outs_g = (B.VerifyOutputs(T), B.VerifyOutputs(T, case.cfg.hidden))
    outs_d = (B.VerifyOutputs(T), B.VerifyOutputs(T, case.cfg.hidden))
    c = case.ctx_len
    gated = 0
    for ctx in (c, c - 37, c - 1, 5, c - 100, c):
        for kv in (kv_g, kv_d):   # every call starts from the committed cache
            for l in range(case.cfg.n_layers):
                kv.k[l].copy_(snap[0][l])
                kv.v[l].copy_(snap[1][l])
        g = run(graph_model, kv_g, ctx, case.tokens, case.parent, outs=outs_g)
        d = run(direct, kv_d, ctx, case.tokens, case.parent, outs=outs_d)
        assert np.array_equal(g["final_hidden"], d["final_hidden"]), ctx
        assert np.array_equal(g["argmax"], d["argmax"]) and np.array_equal(g["top1"], d["top1"]), ctx
        assert g["accepted_nodes"] == d["accepted_nodes"] and g["bonus"] == d["bonus"], ctx
        for l in range(case.cfg.n_layers):
            assert np.array_equal(g["tree_k"][l], d["tree_k"][l]) and np.array_equal(g["tree_v"][l], d["tree_v"][l])
        r = oracle.verify_tree(case.view, [k[:ctx] for k in case.cache_k64], [v[:ctx] for v in case.cache_v64], ctx,
                               case.tokens, case.parent)
        gated += check_case(case, g, r)
    assert gated >= 3


# ------------------------------------------------------------------ accept walk and compaction alone

def test_accept_walk_hand_fixtures_and_random():
    with open(os.path.join(GOLDEN, "accept_cases.json")) as f:
        fixtures = json.load(f)["cases"]
    rng = np.random.default_rng(0)
    cases = [(c["tokens"], c["parent"], c["argmax"]) for c in fixtures]
    for k in range(200):
        T = int(rng.integers(1, 129))
        tokens, parent = trees.random_tokens_tree(T, 1000, key=1000 + k)
        # the greedy token at a node is one of its children's tokens 70% of the time: deep accepted paths
        argmax = rng.integers(0, 1000, size=T)
        for p in range(T):
            kids = [i for i in range(1, T) if parent[i] == p]
            if kids and rng.random() < 0.7:
                argmax[p] = tokens[kids[int(rng.integers(0, len(kids)))]]
        cases.append((tokens.tolist(), parent.tolist(), argmax.tolist()))
    cases.append(([1, 2], [0, 0], [0, 0]))          # malformed
    for tokens, parent, argmax in cases:
        T = len(tokens)
        d = lambda x: torch.as_tensor(np.asarray(x, np.int32), device="cuda")
        outs = B.VerifyOutputs(T)
        st = torch.zeros(1, dtype=torch.int32, device="cuda")
        B.oos_accept_walk(d(tokens), d(parent), d(argmax), T, outs.accepted_len, outs.accepted_nodes,
                          outs.accepted_tokens, outs.bonus, st)
        torch.cuda.synchronize()
        try:
            a = oracle.accept(tokens, parent, argmax)
        except oracle.TreeError:
            assert st.item() == B.OOS_ETREE and outs.accepted_len.item() == 0
            continue
        assert st.item() == B.OOS_OK
        n = outs.accepted_len.item()
        assert n == a["accepted_len"]
        assert outs.accepted_nodes.cpu().tolist()[:n] == a["accepted_nodes"]
        assert outs.accepted_tokens.cpu().tolist()[:n] == a["accepted_tokens"]
        assert outs.bonus.item() == a["bonus"]


def test_kv_compact_matches_gather(tiny_models):
    case, model = _tiny(tiny_models, 0)
    cfg = case.cfg
    rng = np.random.default_rng(1)
    for ctx, path in [(5, [0, 2, 3]), (0, [0, 1, 2, 3]), (7, [0]), (3, [0, 5, 9, 10, 40, 127]),
                      (11, list(range(0, 128, 2))[:40])]:
        cap = ctx + 128
        k = [torch.as_tensor(rng.normal(size=(cap, cfg.n_kv_heads, cfg.head_dim)).astype(np.float32), device="cuda")
             for _ in range(cfg.n_layers)]
        v = [t * -1.5 for t in k]
        kv = B.KVCache(k, v)
        before_k = [t.cpu().numpy().astype(np.float64) for t in kv.k]
        before_v = [t.cpu().numpy().astype(np.float64) for t in kv.v]
        nodes = torch.full((128,), -1, dtype=torch.int32, device="cuda")
        nodes[:len(path)] = torch.as_tensor(path, dtype=torch.int32)
        ln = torch.tensor([len(path)], dtype=torch.int32, device="cuda")
        B.oos_kv_compact(model, kv, ctx, nodes, ln, 128)
        torch.cuda.synchronize()
        ek, ev = oracle.compact(before_k, before_v, ctx, path)
        for l in range(cfg.n_layers):
            assert np.array_equal(kv.k[l].cpu().numpy().astype(np.float64), ek[l])
            assert np.array_equal(kv.v[l].cpu().numpy().astype(np.float64), ev[l])


# ------------------------------------------------------------------ small bf16 decoder (tensor-core path)

@pytest.fixture(scope="module")
def mini_models():
    return {}


def _mini(mini_models, seed, **kw):
    case = build_case("mini-bf16", seed, **kw)
    key = (seed, tuple(sorted((kw.get("cfg_overrides") or {}).items())), kw.get("gain_std", 0.0))
    if key not in mini_models:
        mini_models[key] = gpu_model(case)
    return case, mini_models[key][0]


def test_mini_bf16_parity_seeds(mini_models):
    """Random weight seeds: every tensor at tolerance, accept outputs exact
    wherever the margin gate holds."""
    gated = 0
    for seed in range(6):
        case, model = _mini(mini_models, seed)
        kv = gpu_cache(case, case.ctx_len + 128)
        g = run(model, kv, case.ctx_len, case.tokens, case.parent)
        gated += check_case(case, g, _oracle(case))
        check_compaction(model, kv, case.ctx_len, g)
    assert gated >= 1


def _gated_roots_sweep(name, base, model, min_gated):
    """One case per stored well-separated root (golden/gated_roots.json):
    the workload's tree recipe around root -> greedy path, every node checked
    against the full oracle step; counts the cases whose accept outputs were
    compared exactly (the margin gate)."""
    roots = load_gated_roots(name)
    gated, n = 0, 0
    for k, e in enumerate(roots["cases"]):
        case = with_tree(base, name, e["root"], e["planted"], e["margins"], e["root_index"])
        kv = gpu_cache(case, case.ctx_len + len(case.tokens))
        g = run(model, kv, case.ctx_len, case.tokens, case.parent)
        r = _oracle(case)
        ok = check_case(case, g, r)
        check_compaction(model, kv, case.ctx_len, g)
        if ok:
            assert g["accepted_len"] >= len(case.planted_path)
        gated += ok
        n += 1
    print("%s: %d of %d cases gated (accept outputs compared exactly)" % (name, gated, n))
    assert gated >= min_gated, "%s: only %d of %d cases passed the margin gate" % (name, gated, n)


def test_mini_bf16_gated_roots(mini_models):
    base, model = _mini(mini_models, 0)
    _gated_roots_sweep("mini-bf16", base, model, 20)


def test_mini_f16_cache_gated_roots():
    """The FP16 KV cache (binary16 K/V under bf16 weights): 24 trees around
    well-separated greedy paths of the FP16-cache model, every node against
    the full oracle step."""
    base = build_case("mini-f16", 0)
    model, _ = gpu_model(base)
    _gated_roots_sweep("mini-f16", base, model, 20)


def test_bf16_qwen3_06b_gated_roots():
    """Full-size Qwen3-0.6B shape: 24 trees around well-separated greedy paths,
    every node of every tree against the full oracle step."""
    p = load_planted("qwen3-0.6b")
    base = build_case("qwen3-0.6b", p["seed"], planted=(p["planted"], p["margins"]), root=p["root"])
    model, _ = gpu_model(base)
    _gated_roots_sweep("qwen3-0.6b", base, model, 20)


@pytest.mark.parametrize("T,recipe,ctx", [
    (1, dict(kind="chain"), 200),
    (7, dict(kind="uniform", max_depth=4), 200),        # N tile 16, ragged
    (29, dict(kind="branch", bmin=1, bmax=4, max_depth=8), 200),   # N tile 32
    (50, dict(kind="uniform", max_depth=12), 200),       # N tile 64
    (128, dict(kind="branch", bmin=1, bmax=3, max_depth=30), 200),  # N tile 128, two tree tiles
    (100, dict(kind="chain"), 200),
    (12, dict(kind="uniform", max_depth=5), 0),          # empty cache
    (12, dict(kind="uniform", max_depth=5), 65),         # cache one key past a tile
    (33, dict(kind="uniform", max_depth=8), 4600),       # ~9 tiles per attention block: the K/V ring wraps
])
def test_mini_bf16_shapes(mini_models, T, recipe, ctx):
    case, model = _mini(mini_models, 1, T=T, recipe=recipe, ctx_len=ctx, plant=min(3, T - 1))
    kv = gpu_cache(case, ctx + T)
    g = run(model, kv, ctx, case.tokens, case.parent)
    check_case(case, g, _oracle(case))
    check_compaction(model, kv, ctx, g)


@pytest.mark.parametrize("overrides,gain_std", [(dict(qk_norm=False, qkv_bias=True), 0.2),
                                                (dict(tied=True), 0.1),
                                                (dict(qk_norm=False, rope_factor=8.0, rope_orig_max_pos=256), 0.0)])
def test_mini_bf16_variants(mini_models, overrides, gain_std):
    case, model = _mini(mini_models, 2, cfg_overrides=overrides, gain_std=gain_std)
    kv = gpu_cache(case, case.ctx_len + 16)
    g = run(model, kv, case.ctx_len, case.tokens, case.parent)
    check_case(case, g, _oracle(case))


@pytest.mark.parametrize("T,recipe,ctx", [
    (7, dict(kind="uniform", max_depth=4), 200),
    (50, dict(kind="uniform", max_depth=12), 65),
    (128, dict(kind="branch", bmin=1, bmax=3, max_depth=30), 4600),
    (12, dict(kind="uniform", max_depth=5), 0),
])
def test_mini_f16_cache_shapes(mini_models, T, recipe, ctx):
    """FP16 KV cache under bf16 weights (the paper's Qwen2.5 / Llama backend):
    the cache, the tree's K/V and the attention operands are binary16."""
    case, model = _mini(mini_models, 1, T=T, recipe=recipe, ctx_len=ctx, plant=min(3, T - 1),
                        cfg_overrides=dict(cache_dtype="f16"))
    kv = gpu_cache(case, ctx + T)
    assert kv.k[0].dtype == torch.float16
    g = run(model, kv, ctx, case.tokens, case.parent)
    check_case(case, g, _oracle(case))
    check_compaction(model, kv, ctx, g)


def test_mini_f16_cache_gated_seeds(mini_models):
    gated = 0
    for seed in range(4):
        case, model = _mini(mini_models, seed, cfg_overrides=dict(cache_dtype="f16"))
        kv = gpu_cache(case, case.ctx_len + 16)
        g = run(model, kv, case.ctx_len, case.tokens, case.parent)
        gated += check_case(case, g, _oracle(case))
    assert gated >= 1


def test_fp16_cache_rejected_for_fp32_models():
    case = build_case("tiny", 0, cfg_overrides=dict(cache_dtype="f16"))
    with pytest.raises(B.OosError) as e:
        gpu_model(case)
    assert e.value.code == B.OOS_EUNSUPPORTED


# ------------------------------------------------------------------ bf16 decoders at the workload shapes

def _bf16_case(name, T=None, ctx=None):
    p = load_planted(name)
    return build_case(name, p["seed"], planted=(p["planted"], p["margins"]), T=T, ctx_len=ctx, root=p["root"])


@pytest.mark.parametrize("name", ["qwen3-0.6b", "qwen3-8b"])
def test_bf16_full_size_every_node(name):
    """Full-size parity: every node, every layer, at the workload's shape
    (qwen3-8b: the benchmark's own workload, T=64 over 2048 cached positions)."""
    case = _bf16_case(name)
    model, _ = gpu_model(case)
    kv = gpu_cache(case, case.ctx_len + case.tokens.shape[0])
    g = run(model, kv, case.ctx_len, case.tokens, case.parent)
    r = _oracle(case)
    gated = check_case(case, g, r)
    check_compaction(model, kv, case.ctx_len, g)
    assert gated, "planted path not gated: margins %s" % (r["top1"] - r["top2"])
    assert g["accepted_len"] >= len(case.planted_path)


def _sampled_check(name):
    """Bench-shape parity on sampled nodes: the planted path (and any other
    accepted node) plus two random leaves, with all their ancestors."""
    case = _bf16_case(name)
    model, _ = gpu_model(case)
    kv = gpu_cache(case, case.ctx_len + case.tokens.shape[0])
    g = run(model, kv, case.ctx_len, case.tokens, case.parent)
    T = len(case.tokens)
    leaves = [i for i in range(T) if i not in set(case.parent[1:].tolist())]
    rng = np.random.default_rng(7)
    sample = [case.planted_path[-1]] + list(rng.choice(leaves, size=2, replace=False))
    r = _oracle(case, only=sample)
    rows = r["nodes"]
    # the oracle-accepted set must lie inside the computed rows for the exact check
    computed = set(rows)
    argmax_known = np.where(np.isin(np.arange(T), rows), r["argmax"], -1)
    okn = ok_nodes(case.tokens, case.parent, argmax_known)
    assert set(okn) <= computed
    gated = check_case(case, g, r, rows=rows)
    check_compaction(model, kv, case.ctx_len, g)
    assert gated
    assert g["accepted_len"] == len(case.planted_path) and g["accepted_nodes"] == \
        case.planted_path + [-1] * (T - len(case.planted_path))
    return g


def test_bf16_qwen3_8b_bench_shape_sampled():
    _sampled_check("qwen3-8b")


def test_bf16_llama31_8b_wide_tree_sampled():
    """T=128 wide tree over an 8192-position cache (RoPE theta 5e5 with the
    Llama-3.1 frequency rescaling, no q/k norm)."""
    _sampled_check("llama3.1-8b")


@pytest.mark.parametrize("name", ["qwen3-4b", "qwen3-14b"])
def test_bf16_qwen3_scaling_targets_sampled(name):
    """Qwen3 targets of the paper's scaling study: 4B (tied head, q width 4096
    over hidden 2560) and 14B (40/8 heads, hidden 5120)."""
    _sampled_check(name)


def test_llama31_8b_fp16_cache_sampled():
    """Llama-3.1-8B shape with the FP16 cache the paper runs it with: T=128 wide
    tree over 8192 cached binary16 positions, sampled nodes against the oracle
    (tensors at tolerance, argmax and accept outputs where the margins gate)."""
    p = load_planted("llama3.1-8b")
    case = build_case("llama3.1-8b", p["seed"], planted=(p["planted"], p["margins"]), root=p["root"],
                      cfg_overrides=dict(cache_dtype="f16"))
    model, _ = gpu_model(case)
    kv = gpu_cache(case, case.ctx_len + case.tokens.shape[0])
    assert kv.k[0].dtype == torch.float16
    g = run(model, kv, case.ctx_len, case.tokens, case.parent)
    T = len(case.tokens)
    leaves = [i for i in range(T) if i not in set(case.parent[1:].tolist())]
    rng = np.random.default_rng(9)
    sample = [case.planted_path[-1]] + list(rng.choice(leaves, size=2, replace=False))
    r = _oracle(case, only=sample)
    check_case(case, g, r, rows=r["nodes"])
    check_compaction(model, kv, case.ctx_len, g)


def test_bf16_qwen3_32b_sampled():
    """Qwen3-32B shape of the paper's scaling study (64 layers, hidden 5120,
    64/8 heads, q/k norm, SwiGLU 25600; about 63 GB of bf16 weights): the
    planted path and two leaves, with their ancestors, against the oracle."""
    _sampled_check("qwen3-32b")


def test_bf16_qwen25_32b_sampled():
    """64 layers, 40/8 heads, q/k/v bias: about 64 GB of bf16 weights on one GPU."""
    _sampled_check("qwen2.5-32b")


@pytest.mark.parametrize("name,ctx,n", [
    ("tiny", 0, 300),          # empty cache, three chains of at most 128 tokens (the last one ragged)
    ("tiny", 128, 129),        # after a cached prefix; one full chain and a one-token chain
    ("mini-bf16", 200, 290),   # bf16 tensor-core path
    ("mini-bf16", 0, 1),       # one-token prompt
    ("mini-f16", 200, 150),    # FP16 KV cache
])
def test_prefill_matches_causal_decoding(tiny_models, mini_models, name, ctx, n):
    """oos_prefill == causal decoding of the prompt after ctx cached positions:
    every layer's K/V of the prompt positions, and the greedy next token (when
    its margin clears the gate)."""
    if name == "tiny":
        case, model = _tiny(tiny_models, 4, ctx_len=ctx)
    elif name == "mini-f16":
        case, model = _mini(mini_models, 4, ctx_len=ctx, cfg_overrides=dict(cache_dtype="f16"))
    else:
        case, model = _mini(mini_models, 4, ctx_len=ctx)
    cfg = case.cfg
    prompt = np.random.default_rng(11 + n).integers(0, cfg.vocab, size=n)
    kv = gpu_cache(case, ctx + n + 8)
    tok = torch.as_tensor(prompt.astype(np.int32), device="cuda")
    nxt = torch.full((1,), -1, dtype=torch.int32, device="cuda")
    B.oos_prefill(model, kv, ctx, tok, n, nxt)
    torch.cuda.synchronize()
    assert B.oos_last_status(model) == B.OOS_OK
    steps, ck, cv = oracle.decode_sequence(case.view, case.cache_k64, case.cache_v64, ctx, prompt.tolist())
    tol = TOL[cfg.dtype]
    for l in range(cfg.n_layers):
        ek = max_rel_err(to_f64(cfg, kv.k[l][ctx:ctx + n]), ck[l][ctx:ctx + n])
        ev = max_rel_err(to_f64(cfg, kv.v[l][ctx:ctx + n]), cv[l][ctx:ctx + n])
        assert ek <= tol and ev <= tol, "layer %d prompt K/V error %.3g/%.3g" % (l, ek, ev)
    last = steps[-1]
    if last["top1"] - last["top2"] > GATE[cfg.dtype]:
        assert int(nxt.item()) == int(last["argmax"])
    # the cached prefix is left as it was
    if ctx:
        np.testing.assert_array_equal(to_f64(cfg, kv.k[0][:ctx]), to_f64(cfg, gpu_cache(case, ctx).k[0][:ctx]))
