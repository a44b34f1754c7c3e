"""Random-init decoder weights and KV contents, drawn from seeded streams.

Every tensor is a counter-based stream keyed by (seed, tensor kind, layer), so
the same element can be produced for the GPU (native bf16 / fp32 bits) and for
the fp64 checker (the same values widened exactly) without sharing buffers.

Reading of the initialisation (the paper gives none): matrices, embeddings and
the optional q/k/v biases have mean 0 and std `init_std` (0.02); all RMSNorm
gains are 1 unless `gain_std` > 0 (a test-only variant that jitters them).
Synthetic KV caches hold post-RoPE K and V with mean 0 and std 1.
"""

import numpy as np

from . import gen

# tensor kinds (stream ids)
EMBED, LM_HEAD, FINAL_NORM = 1, 2, 3
ATTN_NORM, W_Q, W_K, W_V, B_Q, B_K, B_V, Q_NORM, K_NORM = 10, 11, 12, 13, 14, 15, 16, 17, 18
W_O, MLP_NORM, W_GATE, W_UP, W_DOWN = 19, 20, 21, 22, 23
KV_K, KV_V = 30, 31
PROMPT, ROOT, TREE_TOKENS, TREE_SHAPE = 40, 41, 42, 43

LAYER_TENSORS = ("attn_norm", "w_q", "w_k", "w_v", "b_q", "b_k", "b_v", "q_norm",
                 "k_norm", "w_o", "mlp_norm", "w_gate", "w_up", "w_down")


class SynthModel:
    """Shapes and streams of one random-init decoder (weights only)."""

    def __init__(self, cfg, seed=0, gain_std=0.0):
        self.cfg = cfg
        self.seed = int(seed)
        self.gain_std = float(gain_std)

    # -- tensor catalogue -------------------------------------------------
    def spec(self, name, layer=0):
        """(kind, shape, sigma, is_gain) of one tensor, or None if absent."""
        c = self.cfg
        H, d, I = c.hidden, c.head_dim, c.intermediate
        s = c.init_std
        table = {
            "embed": (EMBED, (c.vocab, H), s, False),
            "lm_head": (EMBED if c.tied else LM_HEAD, (c.vocab, H), s, False),
            "final_norm": (FINAL_NORM, (H,), None, True),
            "attn_norm": (ATTN_NORM, (H,), None, True),
            "w_q": (W_Q, (c.q_dim, H), s, False),
            "w_k": (W_K, (c.kv_dim, H), s, False),
            "w_v": (W_V, (c.kv_dim, H), s, False),
            "b_q": (B_Q, (c.q_dim,), s, False) if c.qkv_bias else None,
            "b_k": (B_K, (c.kv_dim,), s, False) if c.qkv_bias else None,
            "b_v": (B_V, (c.kv_dim,), s, False) if c.qkv_bias else None,
            "q_norm": (Q_NORM, (d,), None, True) if c.qk_norm else None,
            "k_norm": (K_NORM, (d,), None, True) if c.qk_norm else None,
            "w_o": (W_O, (H, c.q_dim), s, False),
            "mlp_norm": (MLP_NORM, (H,), None, True),
            "w_gate": (W_GATE, (I, H), s, False),
            "w_up": (W_UP, (I, H), s, False),
            "w_down": (W_DOWN, (H, I), s, False),
        }
        return table[name]

    def _key(self, kind, layer):
        # embed / lm_head / final_norm are global tensors: layer id 0
        return gen.tensor_key(self.seed, kind, layer)

    def tensor(self, name, layer=0, fmt="native", out=None):
        """One tensor. fmt: "native" (bf16 bits as uint16, or float32) or "f64".

        `out` (optional) is a reusable buffer of the right size and dtype."""
        sp = self.spec(name, layer)
        if sp is None:
            return None
        kind, shape, sigma, is_gain = sp
        if name in ("embed", "lm_head", "final_norm"):
            layer = 0
        n = int(np.prod(shape))
        bf16 = self.cfg.dtype == "bf16"
        if is_gain:
            if self.gain_std > 0:
                v32 = np.float32(1.0) + gen.normal(self._key(kind, layer), n, self.gain_std, "f32")
            else:
                v32 = np.ones(n, np.float32)
            if bf16:
                bits = gen.np_f32_to_bf16_bits(v32)
                out = bits if fmt == "native" else gen.bf16_bits_to_f64(bits)
            else:
                out = v32 if fmt == "native" else v32.astype(np.float64)
            return out.reshape(shape)
        key = self._key(kind, layer)
        if fmt == "native":
            dt = "bf16" if bf16 else "f32"
        else:
            dt = "bf16_f64" if bf16 else "f32_f64"
        flat = None if out is None else out.reshape(-1)
        return gen.normal(key, n, sigma, dt, out=flat).reshape(shape)

    def rows(self, name, ids, fmt="f64"):
        """Selected rows of a 2-D global tensor (embedding lookups)."""
        kind, shape, sigma, _ = self.spec(name)
        key = self._key(kind, 0)
        H = shape[1]
        bf16 = self.cfg.dtype == "bf16"
        out = []
        for r in np.asarray(ids).reshape(-1):
            dt = ("bf16_f64" if bf16 else "f32_f64") if fmt == "f64" else ("bf16" if bf16 else "f32")
            out.append(gen.normal(key, H, sigma, dt, offset=int(r) * H))
        return np.stack(out) if out else np.zeros((0, H))

    def oracle_view(self, lm_block_rows=16384):
        """Adapter giving the checker fp64 arrays on request (see oracle.Model)."""
        return _OracleView(self, lm_block_rows)


class _OracleView:
    def __init__(self, m, lm_block_rows):
        self._m = m
        self.cfg = m.cfg
        self._lm_block_rows = lm_block_rows
        self._bufs = {}

    def layer(self, l):
        """fp64 tensors of layer l.  Buffers are reused from call to call, so
        a returned dict is valid until the next call."""
        out = {}
        for n in LAYER_TENSORS:
            sp = self._m.spec(n, l)
            if sp is None:
                out[n] = None
                continue
            buf = self._bufs.get(n)
            if buf is None:
                buf = self._bufs[n] = np.empty(sp[1], np.float64)
            out[n] = self._m.tensor(n, l, "f64", out=buf)
        return out

    def embed_rows(self, ids):
        return self._m.rows("embed", ids)

    def final_norm(self):
        return self._m.tensor("final_norm", 0, "f64")

    def lm_head_blocks(self):
        kind, (V, H), sigma, _ = self._m.spec("lm_head")
        key = self._m._key(kind, 0)
        dt = "bf16_f64" if self.cfg.dtype == "bf16" else "f32_f64"
        buf = np.empty(self._lm_block_rows * H, np.float64)
        for r0 in range(0, V, self._lm_block_rows):
            r1 = min(V, r0 + self._lm_block_rows)
            n = (r1 - r0) * H
            yield r0, gen.normal(key, n, sigma, dt, offset=r0 * H, out=buf[:n]).reshape(r1 - r0, H)


def synthetic_kv(cfg, seed, layer, n_pos, fmt="native", which="k"):
    """Synthetic committed K or V of one layer: [n_pos, n_kv_heads, head_dim]."""
    kind = KV_K if which == "k" else KV_V
    key = gen.tensor_key(seed, kind, layer)
    n = n_pos * cfg.kv_dim
    if getattr(cfg, "cache_dtype", "") == "f16":
        # fp32 deviates rounded to IEEE binary16 (nearest even): uint16 bits or their fp64 values
        h = gen.normal(key, n, 1.0, "f32").astype(np.float16)
        out = h.view(np.uint16) if fmt == "native" else h.astype(np.float64)
        return out.reshape(n_pos, cfg.n_kv_heads, cfg.head_dim)
    bf16 = cfg.dtype == "bf16"
    if fmt == "native":
        out = gen.normal(key, n, 1.0, "bf16" if bf16 else "f32")
    else:
        out = gen.normal(key, n, 1.0, "bf16_f64" if bf16 else "f32_f64")
    return out.reshape(n_pos, cfg.n_kv_heads, cfg.head_dim)
