"""The seeded input generator: compiled C == NumPy restatement, bit for bit,
and the published SplitMix64 reference outputs."""

import numpy as np

from synth import gen, trees
from synth.configs import WORKLOADS


def test_splitmix64_reference_values():
    # First outputs of SplitMix64 seeded with 1234567 (Vigna's splitmix64.c,
    # the generator's published reference implementation).
    want = [6457827717110365317, 3203168211198807973, 9817491932198370423,
            4593380528125082431, 16408922859458223821]
    got = [gen.stream_at(1234567, i) for i in range(5)]
    assert got == want
    assert [gen.lib().synth_stream_at(1234567, i) for i in range(5)] == want


def test_compiled_matches_numpy_bitwise():
    for seed, kind, layer in [(0, 11, 0), (3, 30, 7), (12345, 2, 0)]:
        k = gen.tensor_key(seed, kind, layer)
        n, off = 50_000, 987_654
        f = gen.normal(k, n, 0.02, "f32", offset=off)
        ref = gen.np_normal_f32(k, n, 0.02, offset=off)
        np.testing.assert_array_equal(f.view(np.uint32), ref.view(np.uint32))
        b = gen.normal(k, n, 0.02, "bf16", offset=off)
        np.testing.assert_array_equal(b, gen.np_f32_to_bf16_bits(ref))
        w = gen.normal(k, n, 0.02, "bf16_f64", offset=off)
        np.testing.assert_array_equal(w, gen.bf16_bits_to_f64(b))
        u = gen.uniform_int(k, n, 151936, offset=off)
        np.testing.assert_array_equal(u, gen.np_uniform_int(k, n, 151936, offset=off))
        assert u.min() >= 0 and u.max() < 151936


def test_moments():
    x = gen.normal(gen.tensor_key(9, 1, 0), 2_000_000, 0.02, "f32").astype(np.float64)
    assert abs(x.mean()) < 1e-4
    assert abs(x.std() - 0.02) < 1e-4
    assert np.abs(x).max() <= 0.02 * 3.4642


def test_tree_recipes():
    for name, w in WORKLOADS.items():
        planted = list(range(100, 100 + w.plant))
        tok, par, path = trees.make_tree(w.tree, w.T, 5, planted, w.model.vocab, 77)
        assert len(tok) == w.T and par[0] == -1
        assert all(0 <= par[i] < i for i in range(1, w.T))
        assert [int(tok[i]) for i in path] == [5] + planted
        assert all(par[path[j]] == path[j - 1] for j in range(1, len(path)))
        depth = [0] * w.T
        for i in range(1, w.T):
            depth[i] = depth[par[i]] + 1
        assert max(depth) <= w.tree.get("max_depth", w.T)
        # siblings carry distinct tokens
        for p in range(w.T):
            kids = [int(tok[i]) for i in range(1, w.T) if par[i] == p]
            assert len(kids) == len(set(kids))
        if w.tree["kind"] == "branch":
            for p in range(w.T):
                assert sum(1 for i in range(1, w.T) if par[i] == p) <= w.tree["bmax"]
    tok, par, path = trees.make_tree(dict(kind="wide", level_branch=8, max_depth=16), 128, 5,
                                     list(range(12)), 128256, 3)
    assert sum(1 for i in range(1, 128) if par[i] == 0) == 8
