"""ctypes binding of include/oos.h (argument marshalling only).

Every function named oos_* here forwards to the C entry point of the same
name in _lib/liboos.so; PyTorch supplies device memory and the stream.  The
library must be built (paper_2608_00814_gb300._build.build()); importing a
missing library raises -- there is no fallback path.
"""

import ctypes
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_lib", "liboos.so")

OOS_OK = 0
OOS_EINVAL = -1
OOS_ECAPACITY = -2
OOS_ECUDA = -3
OOS_ETREE = -4
OOS_ETIMEOUT = -5
OOS_EUNSUPPORTED = -6
OOS_EWORKSPACE = -7
OOS_DTYPE_F32 = 0
OOS_DTYPE_BF16 = 1

MAX_T = 128

c_i32 = ctypes.c_int32
c_vp = ctypes.c_void_p


class OosModelConfig(ctypes.Structure):
    _fields_ = [("n_layers", c_i32), ("hidden", c_i32), ("n_q_heads", c_i32), ("n_kv_heads", c_i32),
                ("head_dim", c_i32), ("intermediate", c_i32), ("vocab", c_i32), ("dtype", c_i32),
                ("qk_norm", c_i32), ("qkv_bias", c_i32), ("rms_eps", ctypes.c_float),
                ("rope_theta", ctypes.c_float), ("max_T", c_i32), ("use_graph", c_i32),
                ("rope_factor", ctypes.c_float), ("rope_low_freq_factor", ctypes.c_float),
                ("rope_high_freq_factor", ctypes.c_float), ("rope_orig_max_pos", c_i32), ("kv_f16", c_i32)]


LAYER_FIELDS = ("attn_norm", "w_q", "w_k", "w_v", "b_q", "b_k", "b_v", "q_norm", "k_norm", "w_o",
                "mlp_norm", "w_gate", "w_up", "w_down")


class OosLayerWeights(ctypes.Structure):
    _fields_ = [(n, c_vp) for n in LAYER_FIELDS]


class OosWeights(ctypes.Structure):
    _fields_ = [("embed", c_vp), ("final_norm", c_vp), ("lm_head", c_vp),
                ("layers", ctypes.POINTER(OosLayerWeights))]


class OosKvCache(ctypes.Structure):
    _fields_ = [("n_layers", c_i32), ("capacity", c_i32), ("k", ctypes.POINTER(c_vp)),
                ("v", ctypes.POINTER(c_vp))]


_lib = None


def lib():
    """The loaded CUDA library; raises if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError("CUDA library %s is missing: run paper_2608_00814_gb300._build.build()" % LIB_PATH)
        L = ctypes.CDLL(LIB_PATH)
        P = ctypes.POINTER
        L.oos_workspace_bytes.argtypes = [P(OosModelConfig)]
        L.oos_workspace_bytes.restype = ctypes.c_size_t
        L.oos_model_create.argtypes = [P(OosModelConfig), P(OosWeights), c_vp, ctypes.c_size_t, P(c_vp)]
        L.oos_model_destroy.argtypes = [c_vp]
        L.oos_tree_verify.argtypes = [c_vp, P(OosKvCache), c_i32, c_vp, c_vp, c_i32, c_vp, c_vp, c_vp, c_vp, c_vp]
        L.oos_tree_verify_debug.argtypes = [c_vp, P(OosKvCache), c_i32, c_vp, c_vp, c_i32, c_vp, c_vp, c_vp, c_vp,
                                            c_vp, c_vp, c_vp, c_vp, c_vp]
        L.oos_kv_compact.argtypes = [c_vp, P(OosKvCache), c_i32, c_vp, c_vp, c_i32, c_vp]
        L.oos_prefill.argtypes = [c_vp, P(OosKvCache), c_i32, c_vp, c_i32, c_vp, c_vp]
        L.oos_hint_workspace_bytes.argtypes = [c_i32]
        L.oos_hint_workspace_bytes.restype = ctypes.c_size_t
        L.oos_hint_tree.argtypes = [c_vp, c_i32, c_i32, c_vp, c_i32, c_vp, c_vp, c_i32, c_i32, c_i32, c_i32, c_i32,
                                    c_vp, ctypes.c_size_t, c_vp, c_vp, c_vp, c_vp, c_vp]
        L.oos_hint_tree.restype = ctypes.c_int
        L.oos_accept_walk.argtypes = [c_vp, c_vp, c_vp, c_i32, c_vp, c_vp, c_vp, c_vp, c_vp, c_vp]
        L.oos_decode_workspace_bytes.argtypes = [c_i32]
        L.oos_decode_workspace_bytes.restype = ctypes.c_size_t
        L.oos_decode.argtypes = [c_vp, P(OosKvCache), c_i32, c_vp, c_i32, c_i32, c_vp, c_i32, c_i32, c_i32, c_i32,
                                 c_i32, c_i32, c_vp, c_vp, c_vp, ctypes.c_size_t, c_vp]
        L.oos_decode.restype = ctypes.c_int
        L.oos_last_status.argtypes = [c_vp, c_vp]
        L.oos_set_wait_limit.argtypes = [c_vp, ctypes.c_uint64, c_vp]
        L.oos_set_wait_limit.restype = ctypes.c_int
        L.oos_launch_stage.argtypes = [c_vp, c_i32, c_i32, c_i32, c_vp]
        L.oos_launch_stage.restype = ctypes.c_int
        L.oos_launch_attention.argtypes = [c_vp, P(OosKvCache), c_i32, c_i32, c_i32, c_vp]
        L.oos_launch_attention.restype = ctypes.c_int
        L.oos_lm_head_argmax_static.argtypes = [c_i32, c_i32, c_i32, c_vp, c_vp, c_i32, c_vp, c_vp, c_vp, c_vp]
        L.oos_lm_head_argmax_static.restype = ctypes.c_int
        L.oos_status_string.argtypes = [ctypes.c_int]
        L.oos_status_string.restype = ctypes.c_char_p
        for fn in ("oos_model_create", "oos_model_destroy", "oos_tree_verify", "oos_tree_verify_debug",
                   "oos_kv_compact", "oos_accept_walk", "oos_last_status", "oos_prefill"):
            getattr(L, fn).restype = ctypes.c_int
        _lib = L
    return _lib


class OosError(RuntimeError):
    def __init__(self, code, what):
        super().__init__("%s: %s (%d)" % (what, lib().oos_status_string(code).decode(), code))
        self.code = code


def _check(code, what):
    if code != OOS_OK:
        raise OosError(code, what)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def make_config(cfg, max_T, use_graph=True):
    """oos_model_config from an object with the synth ModelConfig fields."""
    return OosModelConfig(cfg.n_layers, cfg.hidden, cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim,
                          cfg.intermediate, cfg.vocab,
                          OOS_DTYPE_BF16 if cfg.dtype == "bf16" else OOS_DTYPE_F32,
                          int(cfg.qk_norm), int(cfg.qkv_bias), cfg.rms_eps, cfg.rope_theta, max_T,
                          int(use_graph), float(getattr(cfg, "rope_factor", 0.0) or 0.0),
                          float(getattr(cfg, "rope_low_freq_factor", 1.0)),
                          float(getattr(cfg, "rope_high_freq_factor", 4.0)),
                          int(getattr(cfg, "rope_orig_max_pos", 8192)),
                          int(getattr(cfg, "cache_dtype", "") == "f16"))


def oos_workspace_bytes(c_cfg):
    return lib().oos_workspace_bytes(ctypes.byref(c_cfg))


class KVCache:
    """Per-layer K and V device tensors [capacity, nkv, d] plus the C view."""

    def __init__(self, k, v):
        assert len(k) == len(v) and len(k) > 0
        self.k, self.v = list(k), list(v)
        self.capacity = k[0].shape[0]
        n = len(k)
        self._kp = (c_vp * n)(*[t.data_ptr() for t in self.k])
        self._vp = (c_vp * n)(*[t.data_ptr() for t in self.v])
        self.c = OosKvCache(n, self.capacity, ctypes.cast(self._kp, ctypes.POINTER(c_vp)),
                            ctypes.cast(self._vp, ctypes.POINTER(c_vp)))

    @staticmethod
    def empty(cfg, capacity, device="cuda"):
        dt = torch.float16 if getattr(cfg, "cache_dtype", "") == "f16" else \
            (torch.bfloat16 if cfg.dtype == "bf16" else torch.float32)
        k = [torch.zeros(capacity, cfg.n_kv_heads, cfg.head_dim, dtype=dt, device=device) for _ in range(cfg.n_layers)]
        v = [torch.zeros_like(t) for t in k]
        return KVCache(k, v)


class OosModel:
    """A model handle: weight pointers, workspace and TMA descriptors.

    weights: dict with "embed", "final_norm", "lm_head" and "layers" (a list of
    dicts keyed by LAYER_FIELDS; absent optional entries may be None), all
    device tensors in the model dtype.  The tensors must outlive the handle.
    """

    def __init__(self, cfg, weights, max_T=MAX_T, use_graph=True):
        self.cfg = cfg
        self.c_cfg = make_config(cfg, max_T, use_graph)
        self.weights = weights
        L = weights["layers"]
        self._layers = (OosLayerWeights * len(L))()
        for i, lw in enumerate(L):
            for n in LAYER_FIELDS:
                t = lw.get(n)
                setattr(self._layers[i], n, None if t is None else t.data_ptr())
        self._w = OosWeights(weights["embed"].data_ptr(), weights["final_norm"].data_ptr(),
                             weights["lm_head"].data_ptr(), self._layers)
        nbytes = oos_workspace_bytes(self.c_cfg)
        if nbytes == 0:
            raise OosError(OOS_EINVAL, "oos_workspace_bytes")
        self.workspace = torch.empty(nbytes + 256, dtype=torch.uint8, device="cuda")
        base = self.workspace.data_ptr()
        self._ws_ptr = (base + 255) // 256 * 256
        h = c_vp()
        _check(lib().oos_model_create(ctypes.byref(self.c_cfg), ctypes.byref(self._w), c_vp(self._ws_ptr), nbytes,
                                      ctypes.byref(h)), "oos_model_create")
        self.handle = h

    def close(self):
        if getattr(self, "handle", None):
            lib().oos_model_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def oos_tree_verify(model, kv, ctx_len, tree_tokens, tree_parent, T, out_accepted_len, out_accepted_nodes,
                    out_accepted_tokens, out_bonus_token, stream=None):
    _check(lib().oos_tree_verify(model.handle, ctypes.byref(kv.c), ctx_len, _ptr(tree_tokens), _ptr(tree_parent), T,
                                 _ptr(out_accepted_len), _ptr(out_accepted_nodes), _ptr(out_accepted_tokens),
                                 _ptr(out_bonus_token), _stream(stream)), "oos_tree_verify")


def oos_tree_verify_debug(model, kv, ctx_len, tree_tokens, tree_parent, T, out_accepted_len, out_accepted_nodes,
                          out_accepted_tokens, out_bonus_token, out_final_hidden=None, out_argmax=None,
                          out_top1=None, out_top2=None, stream=None):
    _check(lib().oos_tree_verify_debug(model.handle, ctypes.byref(kv.c), ctx_len, _ptr(tree_tokens),
                                       _ptr(tree_parent), T, _ptr(out_accepted_len), _ptr(out_accepted_nodes),
                                       _ptr(out_accepted_tokens), _ptr(out_bonus_token), _ptr(out_final_hidden),
                                       _ptr(out_argmax), _ptr(out_top1), _ptr(out_top2), _stream(stream)),
           "oos_tree_verify_debug")


def oos_hint_workspace_bytes(bank_len):
    return int(lib().oos_hint_workspace_bytes(bank_len))


def oos_hint_tree(bank, eos, prefix, native, native_len, max_lanes, depth, max_nodes, workspace, out_tokens,
                  out_parent, out_T, out_info, stream=None):
    """native: int32 [n_native, stride] device tensor (or None), native_len: int32 [n_native]."""
    n_native = 0 if native is None else int(native.shape[0])
    stride = 1 if native is None else int(native.shape[1])
    _check(lib().oos_hint_tree(_ptr(bank), int(bank.numel()), eos, _ptr(prefix), int(prefix.numel()), _ptr(native),
                               _ptr(native_len), n_native, stride, max_lanes, depth, max_nodes, _ptr(workspace),
                               workspace.numel() * workspace.element_size(), _ptr(out_tokens), _ptr(out_parent),
                               _ptr(out_T), _ptr(out_info), _stream(stream)), "oos_hint_tree")


def oos_decode_workspace_bytes(bank_len):
    return int(lib().oos_decode_workspace_bytes(bank_len))


def oos_decode(model, kv, ctx_len, committed, committed_len, bank, eos, max_lanes, depth, max_nodes, n_rounds,
               out_mat, out_state, workspace, stream=None):
    """committed: int32 device tensor (its size is the capacity); bank: int32 device tensor."""
    _check(lib().oos_decode(model.handle, ctypes.byref(kv.c), ctx_len, _ptr(committed), committed_len,
                            int(committed.numel()), _ptr(bank), int(bank.numel()), eos, max_lanes, depth, max_nodes,
                            n_rounds, _ptr(out_mat), _ptr(out_state), _ptr(workspace),
                            workspace.numel() * workspace.element_size(), _stream(stream)), "oos_decode")


def oos_prefill(model, kv, ctx_len, tokens, n, out_next_token=None, stream=None):
    _check(lib().oos_prefill(model.handle, ctypes.byref(kv.c), ctx_len, _ptr(tokens), n, _ptr(out_next_token),
                             _stream(stream)), "oos_prefill")


def oos_kv_compact(model, kv, ctx_len, accepted_nodes, accepted_len, max_len, stream=None):
    _check(lib().oos_kv_compact(model.handle, ctypes.byref(kv.c), ctx_len, _ptr(accepted_nodes), _ptr(accepted_len),
                                max_len, _stream(stream)), "oos_kv_compact")


def oos_accept_walk(tree_tokens, tree_parent, argmax, T, out_accepted_len, out_accepted_nodes, out_accepted_tokens,
                    out_bonus_token, out_status, stream=None):
    _check(lib().oos_accept_walk(_ptr(tree_tokens), _ptr(tree_parent), _ptr(argmax), T, _ptr(out_accepted_len),
                                 _ptr(out_accepted_nodes), _ptr(out_accepted_tokens), _ptr(out_bonus_token),
                                 _ptr(out_status), _stream(stream)), "oos_accept_walk")


OOS_STAGE_QKV, OOS_STAGE_O, OOS_STAGE_GATE_UP, OOS_STAGE_DOWN, OOS_STAGE_LM_HEAD = 0, 1, 2, 3, 4


def oos_launch_stage(model, layer, stage, T, stream=None):
    _check(lib().oos_launch_stage(model.handle, layer, stage, T, _stream(stream)), "oos_launch_stage")


def oos_launch_attention(model, kv, layer, ctx_len, T, stream=None):
    _check(lib().oos_launch_attention(model.handle, ctypes.byref(kv.c), layer, ctx_len, T, _stream(stream)),
           "oos_launch_attention")


def oos_lm_head_argmax_static(dtype, vocab, hidden_dim, lm_head, hidden, T, out_argmax, out_top1, out_top2,
                              stream=None):
    """LM-head greedy argmax that allocates no device memory (see include/oos.h)."""
    _check(lib().oos_lm_head_argmax_static(dtype, vocab, hidden_dim, _ptr(lm_head), _ptr(hidden), T, _ptr(out_argmax),
                                           _ptr(out_top1), _ptr(out_top2), _stream(stream)),
           "oos_lm_head_argmax_static")


def oos_set_wait_limit(model, limit_ns, stream=None):
    _check(lib().oos_set_wait_limit(model.handle, int(limit_ns), _stream(stream)), "oos_set_wait_limit")


def oos_last_status(model, stream=None):
    return lib().oos_last_status(model.handle, _stream(stream))


def oos_status_string(code):
    return lib().oos_status_string(code).decode()


class VerifyOutputs:
    """Device output buffers of one verify call (sized for max_T)."""

    def __init__(self, T, hidden=None, device="cuda"):
        i32 = dict(dtype=torch.int32, device=device)
        self.accepted_len = torch.zeros(1, **i32)
        self.accepted_nodes = torch.zeros(T, **i32)
        self.accepted_tokens = torch.zeros(T, **i32)
        self.bonus = torch.zeros(1, **i32)
        self.final_hidden = None if hidden is None else torch.zeros(T, hidden, dtype=torch.float32, device=device)
        self.argmax = torch.zeros(T, **i32)
        self.top1 = torch.zeros(T, dtype=torch.float32, device=device)
        self.top2 = torch.zeros(T, dtype=torch.float32, device=device)


def tree_verify(model, kv, ctx_len, tokens, parent, outs=None, debug=False, stream=None):
    """Convenience wrapper: verify one tree, return the output buffers."""
    T = int(tokens.shape[0])
    if outs is None:
        outs = VerifyOutputs(T, model.cfg.hidden if debug else None)
    if debug:
        oos_tree_verify_debug(model, kv, ctx_len, tokens, parent, T, outs.accepted_len, outs.accepted_nodes,
                              outs.accepted_tokens, outs.bonus, outs.final_hidden, outs.argmax, outs.top1, outs.top2,
                              stream)
    else:
        oos_tree_verify(model, kv, ctx_len, tokens, parent, T, outs.accepted_len, outs.accepted_nodes,
                        outs.accepted_tokens, outs.bonus, stream)
    return outs
