"""Place seeded synthetic inputs in GPU memory (torch tensors).

Each tensor is generated on the host in its storage type into a pinned
staging buffer and copied to the device, so the GPU and the CPU checker see
the same bits.
"""

import numpy as np
import torch

from .model import LAYER_TENSORS

_STAGE_ELEMS = 1 << 26   # 64 Mi elements per staging chunk


class _Stager:
    def __init__(self, bf16):
        self.bf16 = bf16
        self.dt_t = torch.int16 if bf16 else torch.float32
        self.buf = torch.empty(_STAGE_ELEMS, dtype=self.dt_t, pin_memory=True)
        self.np = self.buf.numpy().view(np.uint16 if bf16 else np.float32)

    def tensor(self, gen_chunk, shape, device):
        """gen_chunk(offset, n, out_numpy) fills elements [offset, offset+n)."""
        n = int(np.prod(shape))
        out = torch.empty(n, dtype=torch.bfloat16 if self.bf16 else torch.float32, device=device)
        flat = out.view(torch.int16) if self.bf16 else out
        for off in range(0, n, _STAGE_ELEMS):
            m = min(_STAGE_ELEMS, n - off)
            gen_chunk(off, m, self.np[:m])
            flat[off:off + m].copy_(self.buf[:m], non_blocking=False)
        return out.view(shape)


def upload_model(sm, device="cuda"):
    """Weights dict for paper_2608_00814_gb300.OosModel (the C ABI layout)."""
    from . import gen
    bf16 = sm.cfg.dtype == "bf16"
    st = _Stager(bf16)
    out_dt = "bf16" if bf16 else "f32"

    def big(name, layer=0):
        kind, shape, sigma, is_gain = sm.spec(name, layer)
        if is_gain:
            arr = sm.tensor(name, layer, "native")
            t = torch.from_numpy(arr.view(np.int16) if bf16 else arr)
            return (t.view(torch.bfloat16) if bf16 else t).to(device)
        key = sm._key(kind, 0 if name in ("embed", "lm_head", "final_norm") else layer)
        return st.tensor(lambda off, n, o: gen.normal(key, n, sigma, out_dt, offset=off, out=o), shape, device)

    w = {"embed": big("embed"), "final_norm": big("final_norm")}
    w["lm_head"] = w["embed"] if sm.cfg.tied else big("lm_head")
    layers = []
    for l in range(sm.cfg.n_layers):
        d = {}
        for n in LAYER_TENSORS:
            d[n] = None if sm.spec(n, l) is None else big(n, l)
        layers.append(d)
    w["layers"] = layers
    return w


def upload_cache(cfg, native_layers, capacity, device="cuda"):
    """K and V device tensors [capacity, nkv, d] per layer; slots past the
    given prefix are zero."""
    f16 = getattr(cfg, "cache_dtype", "") == "f16"
    bf16 = cfg.dtype == "bf16" or f16
    dt = torch.float16 if f16 else (torch.bfloat16 if bf16 else torch.float32)
    ks, vs = [], []
    for k_np, v_np in native_layers:
        n = k_np.shape[0]
        pair = []
        for arr in (k_np, v_np):
            t = torch.zeros(capacity, cfg.n_kv_heads, cfg.head_dim, dtype=dt, device=device)
            if n:
                src = torch.from_numpy(np.ascontiguousarray(arr).view(np.int16) if bf16 else np.ascontiguousarray(arr))
                t[:n].copy_((src.view(dt) if bf16 else src).to(device))
            pair.append(t)
        ks.append(pair[0])
        vs.append(pair[1])
    return ks, vs
