"""Pins of the CPU checker (oracle) against things other than itself.

Library routines (torch.nn.functional, numpy complex arithmetic), closed
forms, brute-force causal decoding along every root-to-leaf path, and
hand-derived fixtures.  No test here needs a GPU.
"""

import dataclasses
import json
import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle
from cases import GOLDEN, build_case
from synth import gen, trees
from synth.configs import TINY
from synth.model import SynthModel



@pytest.fixture(autouse=True)
def _float64_default():
    """fp64 torch defaults for these pins only (restored afterwards, so other
    test modules keep torch's float32 default)."""
    prev = torch.get_default_dtype()
    torch.set_default_dtype(torch.float64)
    yield
    torch.set_default_dtype(prev)


# ------------------------------------------------------------------ tree shape

def test_tree_structure_hand():
    depth, path = oracle.tree_structure([-1, 0, 0, 1, 3, 2])
    assert depth == [0, 1, 1, 2, 3, 2]
    assert path[4] == [0, 1, 3, 4]
    assert path[5] == [0, 2, 5]
    for bad in ([0, 0], [-1, 1], [-1, 0, 2], [-1, -1], [-1, 0, 5], []):
        with pytest.raises(oracle.TreeError):
            oracle.tree_structure(bad)


# ------------------------------------------------------------------ primitives

def test_rms_norm_matches_library_and_closed_form():
    rng = np.random.default_rng(1)
    x = rng.normal(size=(5, 64)) * 3
    g = rng.normal(size=64)
    ref = F.rms_norm(torch.from_numpy(x), (64,), weight=torch.from_numpy(g), eps=1e-6).numpy()
    np.testing.assert_allclose(oracle.rms_norm(x, g, 1e-6), ref, rtol=1e-13, atol=1e-13)
    c = np.full(10, 2.5)
    np.testing.assert_allclose(oracle.rms_norm(c, 1.0, 0.0), np.ones(10), rtol=1e-15)
    np.testing.assert_allclose(oracle.rms_norm(c, 1.0, 1e-2), c / math.sqrt(6.25 + 1e-2), rtol=1e-15)


def test_rope_is_complex_rotation():
    rng = np.random.default_rng(2)
    d, theta = 64, 1e6
    x = rng.normal(size=(3, d))
    for pos in (0, 1, 17, 8191):
        z = x[:, :d // 2] + 1j * x[:, d // 2:]
        inv = 1.0 / theta ** (np.arange(0, d, 2) / d)        # standard frequency table
        zr = z * np.exp(1j * pos * inv)
        ref = np.concatenate([zr.real, zr.imag], axis=-1)
        np.testing.assert_allclose(oracle.rope(x, pos, theta), ref, rtol=1e-12, atol=1e-12)
    np.testing.assert_array_equal(oracle.rope(x, 0, theta), x)


def test_rope_relative_position_and_norm():
    rng = np.random.default_rng(3)
    q, k = rng.normal(size=128), rng.normal(size=128)
    a = oracle.rope(q, 40, 5e5) @ oracle.rope(k, 33, 5e5)
    b = oracle.rope(q, 1040, 5e5) @ oracle.rope(k, 1033, 5e5)
    assert abs(a - b) < 1e-9
    assert abs(np.linalg.norm(oracle.rope(q, 77, 5e5)) - np.linalg.norm(q)) < 1e-12


LLAMA31_ROPE = (8.0, 1.0, 4.0, 8192.0)   # factor, low- and high-frequency factors, original context


def test_rope_rescaling_regions_for_llama31_shape():
    """Llama-3.1 rescaling at theta 5e5, d 128, split by hand.

    Pair m has wavelength 2 pi 5e5^(m/64).  It stays below 8192/4 = 2048 while
    m/64 < ln(2048 / 2 pi) / ln 5e5 = 0.4410, so m <= 28 keep their rate.  It
    exceeds 8192/1 while m/64 > ln(8192 / 2 pi) / ln 5e5 = 0.5467, so m >= 35 turn
    8 times slower.  m = 29..34 are blended.
    """
    base = oracle.rope_inv_freq(128, 5e5)
    np.testing.assert_array_equal(base, 5e5 ** (-np.arange(64) / 64.0))
    r = oracle.rope_inv_freq(128, 5e5, LLAMA31_ROPE) / base
    np.testing.assert_array_equal(r[:29], 1.0)
    np.testing.assert_allclose(r[35:], 1.0 / 8.0, rtol=1e-15)
    mid = r[29:35]
    assert np.all(mid < 1.0) and np.all(mid > 1.0 / 8.0)
    # the blend moves monotonically from the kept rate to the slowed one
    assert np.all(np.diff(r) <= 0.0)


def test_rope_rescaling_blend_is_continuous_at_both_edges():
    """A pair exactly on an edge of the blended band gets the rate of the region
    beyond that edge (the blend weight is 1 at L/hi and 0 at L/lo)."""
    L, lo, hi, F = 8192.0, 1.0, 4.0, 8.0
    for wavelen, want in ((L / hi, 1.0), (L / lo, 1.0 / F)):
        f = 2.0 * np.pi / wavelen
        # theta such that pair m = 1 of d = 4 has rate f: theta^(-1/2) = f
        theta = f ** -2.0
        got = oracle.rope_inv_freq(4, theta, (F, lo, hi, L))[1] / f
        assert abs(got - want) < 1e-12, (wavelen, got, want)


def test_rope_rescaling_none_and_still_a_rotation():
    rng = np.random.default_rng(5)
    q, k = rng.normal(size=128), rng.normal(size=128)
    for sc in (None, (1.0, 1.0, 4.0, 8192.0)):
        # factor <= 1 through the config path means no rescaling at all
        cfg = type("C", (), dict(rope_factor=sc[0] if sc else 0.0, rope_low_freq_factor=1.0,
                                 rope_high_freq_factor=4.0, rope_orig_max_pos=8192))()
        assert oracle.rope_scaling(cfg) is None
    a = oracle.rope(q, 40, 5e5, LLAMA31_ROPE) @ oracle.rope(k, 33, 5e5, LLAMA31_ROPE)
    b = oracle.rope(q, 9040, 5e5, LLAMA31_ROPE) @ oracle.rope(k, 9033, 5e5, LLAMA31_ROPE)
    assert abs(a - b) < 1e-9
    assert abs(np.linalg.norm(oracle.rope(q, 8300, 5e5, LLAMA31_ROPE)) - np.linalg.norm(q)) < 1e-12
    # the slowest pairs turn 8 times less far than without rescaling
    x = np.zeros(128)
    x[63] = 1.0
    ang_scaled = np.arctan2(oracle.rope(x, 1000, 5e5, LLAMA31_ROPE)[127], oracle.rope(x, 1000, 5e5, LLAMA31_ROPE)[63])
    ang_plain = np.arctan2(oracle.rope(x, 1000, 5e5)[127], oracle.rope(x, 1000, 5e5)[63])
    assert abs(ang_scaled * 8.0 - ang_plain) < 1e-12


def test_attend_matches_sdpa():
    rng = np.random.default_rng(4)
    q = rng.normal(size=64)
    K = rng.normal(size=(37, 64))
    V = rng.normal(size=(37, 64))
    ref = F.scaled_dot_product_attention(torch.from_numpy(q)[None, None, None],
                                         torch.from_numpy(K)[None, None],
                                         torch.from_numpy(V)[None, None])[0, 0, 0].numpy()
    np.testing.assert_allclose(oracle.attend(q, K, V), ref, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(oracle.attend(q, K[:1], V[:1]), V[0], rtol=1e-15)


def test_silu_matches_library():
    z = np.linspace(-20, 20, 101)
    np.testing.assert_allclose(oracle.silu(z), F.silu(torch.from_numpy(z)).numpy(), rtol=1e-13, atol=1e-15)


class _Head:
    """Minimal model exposing only an LM head (for argmax pins)."""

    def __init__(self, W, block):
        self.W, self.block = W, block

    def lm_head_blocks(self):
        for r0 in range(0, self.W.shape[0], self.block):
            yield r0, self.W[r0:r0 + self.block]


def test_lm_head_argmax_brute_force_and_ties():
    rng = np.random.default_rng(5)
    W = rng.normal(size=(1000, 16))
    h = rng.normal(size=(4, 16))
    for block in (1000, 128, 7):
        a, t1, t2 = oracle.lm_head_argmax(_Head(W, block), h)
        logits = h @ W.T
        np.testing.assert_array_equal(a, logits.argmax(1))
        srt = np.sort(logits, axis=1)
        np.testing.assert_allclose(t1, srt[:, -1], rtol=0, atol=0)
        np.testing.assert_allclose(t2, srt[:, -2], rtol=0, atol=0)
    # exact ties: duplicated rows on both sides of a block boundary
    W2 = W.copy()
    best = int((h[0] @ W.T).argmax())
    W2[900] = W2[best]
    W2[3] = W2[best]
    for block in (1000, 128, 3):
        a, t1, t2 = oracle.lm_head_argmax(_Head(W2, block), h[:1])
        assert a[0] == min(3, best)
        assert t1[0] == t2[0]


# ------------------------------------------------------------------ accept / compact

def test_accept_hand_fixtures():
    with open(os.path.join(GOLDEN, "accept_cases.json")) as f:
        cases = json.load(f)["cases"]
    for c in cases:
        r = oracle.accept(c["tokens"], c["parent"], c["argmax"])
        for key in ("accepted_len", "accepted_nodes", "accepted_tokens", "bonus"):
            assert r[key] == c[key], (c["note"], key, r[key], c[key])


def test_compact_hazard_is_a_snapshot_gather():
    # path 0 -> 2 -> 3: slot ctx+1 <- ctx+2, slot ctx+2 <- ctx+3 (slot ctx+2 is read before written)
    ctx, cap = 3, 8
    k = np.arange(cap, dtype=np.float64).reshape(cap, 1, 1) * 10
    v = -k
    nk, nv = oracle.compact([k], [v], ctx, [0, 2, 3])
    assert list(nk[0][:, 0, 0]) == [0, 10, 20, 30, 50, 60, 60, 70]
    assert list(nv[0][:, 0, 0]) == [-x for x in [0, 10, 20, 30, 50, 60, 60, 70]]
    assert list(k[:, 0, 0]) == [0, 10, 20, 30, 40, 50, 60, 70]   # inputs untouched


# ------------------------------------------------------------------ whole model: brute force

def _tiny_case(seed, T=8, recipe=None, ctx_len=16, overrides=None, gain_std=0.0, plant=2):
    return build_case("tiny", seed, T=T, recipe=recipe or dict(kind="uniform", max_depth=4),
                      ctx_len=ctx_len, cfg_overrides=overrides, gain_std=gain_std, plant=plant)


@pytest.mark.parametrize("seed", [0, 1])
def test_tree_equals_causal_decoding_on_every_path(seed):
    c = _tiny_case(seed, T=9, overrides=dict(qk_norm=True, qkv_bias=True), gain_std=0.1)
    r = oracle.verify_tree(c.view, c.cache_k64, c.cache_v64, c.ctx_len, c.tokens, c.parent)
    depth, paths = oracle.tree_structure(c.parent)
    leaves = [i for i in range(len(c.parent)) if i not in set(c.parent[1:].tolist())]
    for leaf in leaves:
        path = paths[leaf]
        steps, _, _ = oracle.decode_sequence(c.view, c.cache_k64, c.cache_v64, c.ctx_len,
                                             c.tokens[path])
        for j, node in enumerate(path):
            np.testing.assert_allclose(r["final_hidden"][node], steps[j]["final_hidden"],
                                       rtol=1e-10, atol=1e-10)
            assert r["argmax"][node] == steps[j]["argmax"]
            for l in range(c.cfg.n_layers):
                np.testing.assert_allclose(r["tree_k"][l][node], steps[j]["k"][l], rtol=1e-10, atol=1e-10)
                np.testing.assert_allclose(r["tree_v"][l][node], steps[j]["v"][l], rtol=1e-10, atol=1e-10)


def test_chain_tree_is_causal_decoding():
    c = _tiny_case(3, T=6, recipe=dict(kind="chain"), plant=0)
    r = oracle.verify_tree(c.view, c.cache_k64, c.cache_v64, c.ctx_len, c.tokens, c.parent)
    order = [0]
    while len(order) < 6:
        order.append(int(np.where(c.parent == order[-1])[0][0]))
    steps, _, _ = oracle.decode_sequence(c.view, c.cache_k64, c.cache_v64, c.ctx_len, c.tokens[order])
    for j, node in enumerate(order):
        np.testing.assert_allclose(r["final_hidden"][node], steps[j]["final_hidden"], rtol=1e-10, atol=1e-10)


def test_planted_path_fully_accepted_and_vanilla_step():
    c = _tiny_case(4, T=8, plant=3)
    r = oracle.verify_and_accept(c.view, c.cache_k64, c.cache_v64, c.ctx_len, c.tokens, c.parent)
    assert r["accepted_len"] >= 4
    assert r["accepted_nodes"][:4] == c.planted_path
    # the bonus after the planted path is the next greedy token
    nxt, _ = oracle.greedy_continuation(c.view, c.cache_k64, c.cache_v64, c.ctx_len,
                                        c.tokens[0], r["accepted_len"])
    assert r["bonus"] == nxt[-1]
    # T = 1: one ordinary decode step
    r1 = oracle.verify_and_accept(c.view, c.cache_k64, c.cache_v64, c.ctx_len, c.tokens[:1], [-1])
    hf, a, _, _, _, _ = oracle.decode_step(c.view, c.cache_k64, c.cache_v64, c.ctx_len, int(c.tokens[0]))
    assert r1["accepted_len"] == 1 and r1["bonus"] == a == nxt[0]


def test_random_child_is_rejected():
    c = _tiny_case(5, T=4, recipe=dict(kind="chain"), plant=1)
    r = oracle.verify_tree(c.view, c.cache_k64, c.cache_v64, c.ctx_len, c.tokens, c.parent)
    tokens = c.tokens.copy()
    # node on the chain below the planted child gets a token that is not the greedy one
    child = int(np.where(c.parent == 0)[0][0])
    grand = int(np.where(c.parent == child)[0][0])
    tokens[grand] = (r["argmax"][child] + 1) % c.cfg.vocab
    a = oracle.accept(tokens, c.parent, r["argmax"])
    assert a["accepted_nodes"] == [0, child]
    assert a["bonus"] == r["argmax"][child]


def test_relabelling_invariance():
    c = _tiny_case(6, T=8)
    r = oracle.verify_tree(c.view, c.cache_k64, c.cache_v64, c.ctx_len, c.tokens, c.parent)
    # another topological numbering: sort by (depth, old id)
    depth, _ = oracle.tree_structure(c.parent)
    order = sorted(range(8), key=lambda i: (depth[i], i))
    new = {old: n for n, old in enumerate(order)}
    tok2 = np.array([c.tokens[o] for o in order])
    par2 = np.array([-1 if o == 0 else new[int(c.parent[o])] for o in order])
    r2 = oracle.verify_tree(c.view, c.cache_k64, c.cache_v64, c.ctx_len, tok2, par2)
    for old in range(8):
        np.testing.assert_allclose(r2["final_hidden"][new[old]], r["final_hidden"][old], rtol=1e-11, atol=1e-11)
        assert r2["argmax"][new[old]] == r["argmax"][old]


# ------------------------------------------------------------------ whole model: library restatement

def _torch_tree_forward(m, cfg, prompt, tokens, parent):
    """Independent restatement with torch library ops over prompt + tree.

    Prompt position p sees prompt positions <= p; tree node i sees the whole
    prompt and its ancestors; positions are p and C + depth(i).
    """
    C, T = len(prompt), len(tokens)
    depth, paths = oracle.tree_structure(parent)
    ids = list(prompt) + list(tokens)
    N = C + T
    pos = torch.tensor(list(range(C)) + [C + dd for dd in depth], dtype=torch.float64)
    allow = torch.zeros(N, N, dtype=torch.bool)
    for p in range(C):
        allow[p, :p + 1] = True
    for i in range(T):
        allow[C + i, :C] = True
        for a in paths[i]:
            allow[C + i, C + a] = True
    x = torch.from_numpy(m.embed_rows(ids))
    nq, nkv, d = cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim
    inv_freq = 1.0 / (cfg.rope_theta ** (torch.arange(0, d, 2, dtype=torch.float64) / d))
    rot = torch.polar(torch.ones(N, d // 2), pos[:, None] * inv_freq[None])

    def rope_t(t):                      # t [N, heads, d]
        z = torch.complex(t[..., :d // 2], t[..., d // 2:]) * rot[:, None, :]
        return torch.cat([z.real, z.imag], dim=-1)

    ks, vs = [], []
    for l in range(cfg.n_layers):
        W = {k: (None if v is None else torch.from_numpy(np.array(v))) for k, v in m.layer(l).items()}
        h = F.rms_norm(x, (cfg.hidden,), weight=W["attn_norm"], eps=cfg.rms_eps)
        q = F.linear(h, W["w_q"], W["b_q"]).view(N, nq, d)
        k = F.linear(h, W["w_k"], W["b_k"]).view(N, nkv, d)
        v = F.linear(h, W["w_v"], W["b_v"]).view(N, nkv, d)
        if W["q_norm"] is not None:
            q = F.rms_norm(q, (d,), weight=W["q_norm"], eps=cfg.rms_eps)
            k = F.rms_norm(k, (d,), weight=W["k_norm"], eps=cfg.rms_eps)
        q, k = rope_t(q), rope_t(k)
        ks.append(k)
        vs.append(v)
        kk = k.repeat_interleave(nq // nkv, dim=1)
        vv = v.repeat_interleave(nq // nkv, dim=1)
        o = F.scaled_dot_product_attention(q.transpose(0, 1), kk.transpose(0, 1), vv.transpose(0, 1),
                                           attn_mask=allow)
        x = x + F.linear(o.transpose(0, 1).reshape(N, nq * d), W["w_o"])
        h = F.rms_norm(x, (cfg.hidden,), weight=W["mlp_norm"], eps=cfg.rms_eps)
        x = x + F.linear(F.silu(F.linear(h, W["w_gate"])) * F.linear(h, W["w_up"]), W["w_down"])
    hf = F.rms_norm(x, (cfg.hidden,), weight=torch.from_numpy(m.final_norm()), eps=cfg.rms_eps)
    W_lm = torch.cat([torch.from_numpy(np.array(b)) for _, b in m.lm_head_blocks()])
    logits = F.linear(hf, W_lm)
    return hf.numpy(), logits.argmax(-1).numpy(), [k.numpy() for k in ks], [v.numpy() for v in vs]


@pytest.mark.parametrize("overrides,gain_std", [({}, 0.0),
                                                (dict(qk_norm=True, qkv_bias=True, tied=True), 0.2)])
def test_tree_pass_matches_library_restatement(overrides, gain_std):
    cfg = dataclasses.replace(TINY, **overrides)
    sm = SynthModel(cfg, seed=11, gain_std=gain_std)
    m = sm.oracle_view(lm_block_rows=300)
    C = 12
    prompt = gen.uniform_int(gen.tensor_key(11, 40), C, cfg.vocab)
    tokens, parent = trees.random_tokens_tree(9, cfg.vocab, key=1234)
    hf_t, arg_t, ks_t, vs_t = _torch_tree_forward(m, cfg, prompt, tokens, parent)
    ck, cv, _ = oracle.prefill(m, prompt)
    r = oracle.verify_tree(m, ck, cv, C, tokens, parent)
    np.testing.assert_allclose(r["final_hidden"], hf_t[C:], rtol=1e-10, atol=1e-10)
    np.testing.assert_array_equal(r["argmax"], arg_t[C:])
    for l in range(cfg.n_layers):
        np.testing.assert_allclose(ck[l], ks_t[l][:C], rtol=1e-10, atol=1e-10)
        np.testing.assert_allclose(cv[l], vs_t[l][:C], rtol=1e-10, atol=1e-10)
        np.testing.assert_allclose(r["tree_k"][l], ks_t[l][C:], rtol=1e-10, atol=1e-10)
        np.testing.assert_allclose(r["tree_v"][l], vs_t[l][C:], rtol=1e-10, atol=1e-10)


def test_only_subset_matches_full_pass():
    c = _tiny_case(7, T=8)
    full = oracle.verify_tree(c.view, c.cache_k64, c.cache_v64, c.ctx_len, c.tokens, c.parent)
    leaf = 7
    part = oracle.verify_tree(c.view, c.cache_k64, c.cache_v64, c.ctx_len, c.tokens, c.parent, only=[leaf])
    for i in part["nodes"]:
        np.testing.assert_allclose(part["final_hidden"][i], full["final_hidden"][i], rtol=1e-12, atol=1e-12)
        assert part["argmax"][i] == full["argmax"][i]


# ------------------------------------------------------------------ bf16 KV cache format

def test_cache_format_is_bf16_round_to_nearest_even():
    rng = np.random.default_rng(11)
    x = np.concatenate([rng.standard_normal(4096) * 3.0, [0.0, -0.0, 1.0, -2.5, 1e-30, 65504.0]])
    # exact bf16 halfway points (fp32 low half 0x8000), both parities of the kept bit
    halves = (np.arange(64, dtype=np.uint32) << 16 | np.uint32(0x3F800000) | np.uint32(0x8000)).view(np.float32)
    x = np.concatenate([x, halves.astype(np.float64), -halves.astype(np.float64)])
    ref = torch.from_numpy(x).to(torch.float32).to(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(oracle.cache_format(x, "bf16"), ref)
    np.testing.assert_array_equal(oracle.cache_format(x, "f32"), x)


def test_cache_format_f16_round_to_nearest_even():
    """fp16 cache format: hand-worked binary16 cases, then torch's conversion."""
    u = 2.0 ** -11                      # half a unit in the last place at 1.0
    sub = 2.0 ** -24                    # smallest binary16 subnormal
    cases = [(1.0 + u, 1.0),            # tie, kept bit even: down
             (1.0 + 3 * u, 1.0 + 4 * u),  # tie, kept bit odd: up
             (65504.0, 65504.0),        # largest finite
             (65520.0, np.inf),         # tie between 65504 and 2^16: to even, which overflows
             (sub / 2, 0.0),            # tie between 0 and the smallest subnormal: to 0
             (1.5 * sub, 2 * sub),      # tie between 1 and 2 subnormal units: to 2
             (-1.0 - u, -1.0)]
    x = np.array([c[0] for c in cases])
    np.testing.assert_array_equal(oracle.cache_format(x, "f16"), np.array([c[1] for c in cases]))
    rng = np.random.default_rng(12)
    y = rng.standard_normal(4096) * 50.0
    ref = torch.from_numpy(y).to(torch.float32).to(torch.float16).to(torch.float64).numpy()
    np.testing.assert_array_equal(oracle.cache_format(y, "f16"), ref)


def _mini_case(seed, T=7, ctx_len=12):
    return build_case("mini-bf16", seed, T=T, recipe=dict(kind="uniform", max_depth=3), ctx_len=ctx_len, plant=0)


def test_bf16_tree_kv_is_cache_format_and_tree_equals_causal_decoding():
    """With a bf16 cache both the tree pass and plain decoding attend to bf16
    K/V; the tree pass still equals causal decoding along every path."""
    c = _mini_case(5)
    r = oracle.verify_tree(c.view, c.cache_k64, c.cache_v64, c.ctx_len, c.tokens, c.parent)
    for l in range(c.cfg.n_layers):
        np.testing.assert_array_equal(oracle.cache_format(r["tree_k"][l], "bf16"), r["tree_k"][l])
        np.testing.assert_array_equal(oracle.cache_format(r["tree_v"][l], "bf16"), r["tree_v"][l])
    _, paths = oracle.tree_structure(c.parent)
    leaves = [i for i in range(len(c.parent)) if i not in set(c.parent[1:].tolist())]
    for leaf in leaves:
        path = paths[leaf]
        steps, _, _ = oracle.decode_sequence(c.view, c.cache_k64, c.cache_v64, c.ctx_len, c.tokens[path])
        for j, node in enumerate(path):
            np.testing.assert_allclose(r["final_hidden"][node], steps[j]["final_hidden"], rtol=1e-10, atol=1e-10)
            for l in range(c.cfg.n_layers):
                np.testing.assert_array_equal(r["tree_k"][l][node], steps[j]["k"][l])


def test_bf16_layer0_tree_k_matches_library_restatement():
    """Layer-0 K of every node: RMSNorm, W_k, per-head RMSNorm, rotary
    embedding at ctx + depth, then bf16 -- restated with torch routines."""
    c = _mini_case(6)
    r = oracle.verify_tree(c.view, c.cache_k64, c.cache_v64, c.ctx_len, c.tokens, c.parent)
    W = c.view.layer(0)
    cfg = c.cfg
    depth, _ = oracle.tree_structure(c.parent)
    x = torch.from_numpy(c.view.embed_rows(c.tokens))
    h = F.rms_norm(x, (cfg.hidden,), torch.from_numpy(W["attn_norm"]), eps=cfg.rms_eps)
    k = (h @ torch.from_numpy(W["w_k"]).T).reshape(len(c.tokens), cfg.n_kv_heads, cfg.head_dim)
    k = F.rms_norm(k, (cfg.head_dim,), torch.from_numpy(W["k_norm"]), eps=cfg.rms_eps)
    half = cfg.head_dim // 2
    freq = cfg.rope_theta ** (-2.0 * torch.arange(half, dtype=torch.float64) / cfg.head_dim)
    pos = torch.tensor([c.ctx_len + d for d in depth], dtype=torch.float64)
    rot = torch.polar(torch.ones(len(depth), half, dtype=torch.float64), pos[:, None] * freq[None, :])
    kc = torch.complex(k[..., :half], k[..., half:]) * rot[:, None, :]
    k_rot = torch.cat([kc.real, kc.imag], dim=-1)
    ref = k_rot.to(torch.float32).to(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_allclose(r["tree_k"][0], ref, rtol=0, atol=0)


def _mini_f16_case(seed, T=7, ctx_len=12):
    return build_case("mini-bf16", seed, T=T, recipe=dict(kind="uniform", max_depth=3), ctx_len=ctx_len, plant=0,
                      cfg_overrides=dict(cache_dtype="f16"))


def test_f16_cache_tree_kv_and_tree_equals_causal_decoding():
    """FP16 cache (the paper's Qwen2.5 / Llama backend) under bf16 weights: the
    cache and every K/V a node attends to are binary16, the tree pass equals
    causal decoding along every path, and layer-0 K equals the library
    restatement rounded by torch's own fp32 -> fp16 conversion."""
    c = _mini_f16_case(7)
    assert oracle.kv_format(c.cfg) == "f16" and c.cfg.dtype == "bf16"
    for l in range(c.cfg.n_layers):   # the committed cache is binary16 values
        np.testing.assert_array_equal(c.cache_k64[l].astype(np.float16).astype(np.float64), c.cache_k64[l])
    r = oracle.verify_tree(c.view, c.cache_k64, c.cache_v64, c.ctx_len, c.tokens, c.parent)
    for l in range(c.cfg.n_layers):
        np.testing.assert_array_equal(r["tree_k"][l].astype(np.float16).astype(np.float64), r["tree_k"][l])
        np.testing.assert_array_equal(r["tree_v"][l].astype(np.float16).astype(np.float64), r["tree_v"][l])
    _, paths = oracle.tree_structure(c.parent)
    leaves = [i for i in range(len(c.parent)) if i not in set(c.parent[1:].tolist())]
    for leaf in leaves:
        path = paths[leaf]
        steps, _, _ = oracle.decode_sequence(c.view, c.cache_k64, c.cache_v64, c.ctx_len, c.tokens[path])
        for j, node in enumerate(path):
            np.testing.assert_allclose(r["final_hidden"][node], steps[j]["final_hidden"], rtol=1e-10, atol=1e-10)
            for l in range(c.cfg.n_layers):
                np.testing.assert_array_equal(r["tree_k"][l][node], steps[j]["k"][l])
    W = c.view.layer(0)
    cfg = c.cfg
    depth, _ = oracle.tree_structure(c.parent)
    x = torch.from_numpy(c.view.embed_rows(c.tokens))
    h = F.rms_norm(x, (cfg.hidden,), torch.from_numpy(W["attn_norm"]), eps=cfg.rms_eps)
    v = (h @ torch.from_numpy(W["w_v"]).T).reshape(len(c.tokens), cfg.n_kv_heads, cfg.head_dim)
    np.testing.assert_array_equal(r["tree_v"][0], v.to(torch.float32).to(torch.float16).to(torch.float64).numpy())


def test_f16_and_bf16_caches_differ_only_by_the_cache_rounding():
    """Same weights, same tree: the two cache formats give final hiddens that
    differ (the cache rounding changes), but by far less than the bf16
    tolerance."""
    a = _mini_case(9)
    b = _mini_f16_case(9)
    ra = oracle.verify_tree(a.view, a.cache_k64, a.cache_v64, a.ctx_len, a.tokens, a.parent)
    rb = oracle.verify_tree(b.view, b.cache_k64, b.cache_v64, b.ctx_len, b.tokens, b.parent)
    d = np.abs(ra["final_hidden"] - rb["final_hidden"]).max() / max(1.0, np.abs(ra["final_hidden"]).max())
    assert 0.0 < d < 2e-2
