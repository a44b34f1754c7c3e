"""Model shapes and tree-workload recipes for the verify-step workloads.

Five decoder shapes: a tiny fp32 decoder for exhaustive parity checks and four
random-init bf16 decoders shaped like the targets the paper evaluates
(Qwen3-0.6B / Qwen3-8B, Llama-3.1-8B and Qwen2.5-32B; experimental setup,
"Targets, Workloads, and Protocol").  Only shapes live here: no arithmetic of
the method.

Tree recipes follow the paper's accepted lengths (#MAT between 3.86 and 8.71
in the main comparison table): one greedy path of `plant` draft nodes is
planted under the root, the remaining nodes are random draft tokens.
"""

import dataclasses
from dataclasses import dataclass, field, asdict


@dataclass(frozen=True)
class ModelConfig:
    name: str
    n_layers: int
    hidden: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    intermediate: int
    vocab: int
    rms_eps: float
    rope_theta: float
    dtype: str            # "f32" or "bf16": storage type of weights and KV
    qk_norm: bool         # Qwen3: per-head RMSNorm of q and k before RoPE
    qkv_bias: bool        # Qwen2.5: bias on the q, k, v projections
    tied: bool            # LM head shares the embedding matrix
    init_std: float = 0.02
    # element type of the KV cache when it differs from `dtype` ("f16": the
    # FP16 cache backend the paper's Qwen2.5 and Llama runs use); "" = dtype
    cache_dtype: str = ""
    # Llama 3.1 rotary frequency rescaling (factor <= 1: none)
    rope_factor: float = 0.0
    rope_low_freq_factor: float = 1.0
    rope_high_freq_factor: float = 4.0
    rope_orig_max_pos: int = 8192

    @property
    def q_dim(self):
        return self.n_q_heads * self.head_dim

    @property
    def kv_dim(self):
        return self.n_kv_heads * self.head_dim

    @property
    def kv_dtype(self):
        return self.cache_dtype or self.dtype

    def as_dict(self):
        return asdict(self)


@dataclass(frozen=True)
class Workload:
    model: ModelConfig
    ctx_len: int          # committed positions already in the KV cache
    T: int                # tree nodes, root included
    plant: int            # draft nodes on the planted greedy path (below the root)
    tree: dict = field(default_factory=dict)
    prefill: bool = False  # tiny only: the cache holds a real prefill of ctx_len tokens

    @property
    def name(self):
        return self.model.name


TINY = ModelConfig("tiny", n_layers=2, hidden=256, n_q_heads=4, n_kv_heads=2,
                   head_dim=64, intermediate=512, vocab=1024, rms_eps=1e-6,
                   rope_theta=1e6, dtype="f32", qk_norm=False, qkv_bias=False,
                   tied=False)

QWEN3_0_6B = ModelConfig("qwen3-0.6b", n_layers=28, hidden=1024, n_q_heads=16,
                         n_kv_heads=8, head_dim=128, intermediate=3072,
                         vocab=151936, rms_eps=1e-6, rope_theta=1e6,
                         dtype="bf16", qk_norm=True, qkv_bias=False, tied=True)

QWEN3_8B = ModelConfig("qwen3-8b", n_layers=36, hidden=4096, n_q_heads=32,
                       n_kv_heads=8, head_dim=128, intermediate=12288,
                       vocab=151936, rms_eps=1e-6, rope_theta=1e6,
                       dtype="bf16", qk_norm=True, qkv_bias=False, tied=False)

# Qwen3 targets of the paper's scaling study (4B, 8B, 14B, 32B with one frozen sidecar)
QWEN3_4B = ModelConfig("qwen3-4b", n_layers=36, hidden=2560, n_q_heads=32,
                       n_kv_heads=8, head_dim=128, intermediate=9728,
                       vocab=151936, rms_eps=1e-6, rope_theta=1e6,
                       dtype="bf16", qk_norm=True, qkv_bias=False, tied=True)

QWEN3_14B = ModelConfig("qwen3-14b", n_layers=40, hidden=5120, n_q_heads=40,
                        n_kv_heads=8, head_dim=128, intermediate=17408,
                        vocab=151936, rms_eps=1e-6, rope_theta=1e6,
                        dtype="bf16", qk_norm=True, qkv_bias=False, tied=False)

QWEN3_32B = ModelConfig("qwen3-32b", n_layers=64, hidden=5120, n_q_heads=64,
                        n_kv_heads=8, head_dim=128, intermediate=25600,
                        vocab=151936, rms_eps=1e-6, rope_theta=1e6,
                        dtype="bf16", qk_norm=True, qkv_bias=False, tied=False)

LLAMA31_8B = ModelConfig("llama3.1-8b", n_layers=32, hidden=4096, n_q_heads=32,
                         n_kv_heads=8, head_dim=128, intermediate=14336,
                         vocab=128256, rms_eps=1e-5, rope_theta=5e5,
                         dtype="bf16", qk_norm=False, qkv_bias=False, tied=False,
                         rope_factor=8.0, rope_low_freq_factor=1.0, rope_high_freq_factor=4.0,
                         rope_orig_max_pos=8192)

QWEN25_32B = ModelConfig("qwen2.5-32b", n_layers=64, hidden=5120, n_q_heads=40,
                         n_kv_heads=8, head_dim=128, intermediate=27648,
                         vocab=152064, rms_eps=1e-6, rope_theta=1e6,
                         dtype="bf16", qk_norm=False, qkv_bias=True, tied=False)

WORKLOADS = {
    "tiny": Workload(TINY, ctx_len=128, T=8, plant=3,
                     tree=dict(kind="uniform", max_depth=4), prefill=True),
    "qwen3-0.6b": Workload(QWEN3_0_6B, ctx_len=1024, T=32, plant=6,
                           tree=dict(kind="branch", bmin=1, bmax=4, max_depth=8)),
    "qwen3-8b": Workload(QWEN3_8B, ctx_len=2048, T=64, plant=10,
                         tree=dict(kind="branch", bmin=1, bmax=4, max_depth=12)),
    "llama3.1-8b": Workload(LLAMA31_8B, ctx_len=8192, T=128, plant=12,
                            tree=dict(kind="wide", level_branch=8, max_depth=16)),
    "qwen2.5-32b": Workload(QWEN25_32B, ctx_len=4096, T=64, plant=10,
                            tree=dict(kind="branch", bmin=1, bmax=4, max_depth=12)),
    "qwen3-4b": Workload(QWEN3_4B, ctx_len=2048, T=64, plant=10,
                         tree=dict(kind="branch", bmin=1, bmax=4, max_depth=12)),
    "qwen3-14b": Workload(QWEN3_14B, ctx_len=2048, T=64, plant=10,
                          tree=dict(kind="branch", bmin=1, bmax=4, max_depth=12)),
    "qwen3-32b": Workload(QWEN3_32B, ctx_len=2048, T=64, plant=10,
                          tree=dict(kind="branch", bmin=1, bmax=4, max_depth=12)),
}

# A small bf16 decoder with the head_dim of the real targets: runs every
# tensor-core kernel of the bf16 path at sizes the CPU checker finishes in
# seconds (tests and the smoke check only; not a benchmark workload).
MINI_BF16 = ModelConfig("mini-bf16", n_layers=2, hidden=256, n_q_heads=4, n_kv_heads=2,
                        head_dim=128, intermediate=512, vocab=4096, rms_eps=1e-6,
                        rope_theta=1e6, dtype="bf16", qk_norm=True, qkv_bias=False, tied=False,
                        init_std=0.08)

# The same decoder with the FP16 KV cache (binary16 K/V, bf16 weights): the
# cache backend the paper runs Qwen2.5 and Llama with.
MINI_F16 = dataclasses.replace(MINI_BF16, name="mini-f16", cache_dtype="f16")

TEST_WORKLOADS = {
    "mini-bf16": Workload(MINI_BF16, ctx_len=200, T=16, plant=3,
                          tree=dict(kind="uniform", max_depth=6), prefill=True),
    "mini-f16": Workload(MINI_F16, ctx_len=200, T=16, plant=3,
                         tree=dict(kind="uniform", max_depth=6), prefill=True),
}

MODELS = {w.model.name: w.model for w in list(WORKLOADS.values()) + list(TEST_WORKLOADS.values())}


def workload(name):
    return WORKLOADS[name] if name in WORKLOADS else TEST_WORKLOADS[name]


def weight_bytes(cfg: ModelConfig) -> dict:
    """Bytes of every weight tensor class of one model (embedding excluded)."""
    esz = 4 if cfg.dtype == "f32" else 2
    H, I = cfg.hidden, cfg.intermediate
    per_layer = (cfg.q_dim + 2 * cfg.kv_dim) * H + H * cfg.q_dim + 3 * H * I
    small = 2 * H + (2 * cfg.head_dim if cfg.qk_norm else 0) + \
        ((cfg.q_dim + 2 * cfg.kv_dim) if cfg.qkv_bias else 0)
    return dict(layers=cfg.n_layers * (per_layer + small) * esz,
                lm_head=cfg.vocab * H * esz,
                final_norm=H * esz)
