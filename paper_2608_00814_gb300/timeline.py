"""Step timeline of the bf16 verify kernels on one GPU: per-CTA globaltimer
events of every weight-GEMM launch and of the last attention launch of one
graph-replayed step, read from the library built with -DOOS_TIMELINE
(`_build.build(timeline=True)`, a separate .so; the product library has no
stamps).

    python -m paper_2608_00814_gb300.timeline [--workload qwen3-8b] [--layers L]

Printed per GEMM kind (q/k/v, O, gate/up, down), averaged over the layers:
  main     first CTA entry -> the last CTA's last accumulator ready
  tail     last accumulator ready -> last CTA exit, split into publish (-> the
           last arrival count), poll (-> the last finisher released) and
           finish (-> the last exit)
and per layer the time from one kernel's last exit to the next one's
(attention included), then the attention's phases (median over its blocks,
from the earliest block entry).  The stamps cost a few global stores per CTA;
everything else is the product path.  Run from the repository root (the
workload's tree comes from bench.py).
"""

import argparse
import ctypes
import dataclasses
import sys

import numpy as np


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--workload", default="qwen3-8b")
    ap.add_argument("--layers", type=int, default=0, help="first L layers only (0: all)")
    args = ap.parse_args()

    from . import _build
    from . import binding as B
    B.LIB_PATH = _build.build(timeline=True)
    import torch

    sys.path.insert(0, _build.ROOT)
    import bench
    from synth.configs import WORKLOADS
    from synth.device import upload_cache, upload_model
    from synth.model import SynthModel, synthetic_kv

    w = WORKLOADS[args.workload]
    cfg = w.model if not args.layers else dataclasses.replace(w.model, n_layers=args.layers)
    T, ctx = w.T, w.ctx_len
    seed, tok_np, par_np, _ = bench.workload_tree(args.workload)
    weights = upload_model(SynthModel(cfg, seed))
    native = [(synthetic_kv(cfg, seed, l, ctx, "native", "k"), synthetic_kv(cfg, seed, l, ctx, "native", "v"))
              for l in range(cfg.n_layers)]
    k, v = upload_cache(cfg, native, ctx + T)
    kv = B.KVCache(k, v)
    model = B.OosModel(cfg, weights, max_T=T, use_graph=True)
    L = B.lib()
    for f in ("oos_timeline_gemm_read", "oos_timeline_attn_read"):
        getattr(L, f).argtypes = [ctypes.c_void_p, ctypes.c_size_t]
    tok = torch.as_tensor(tok_np, dtype=torch.int32, device="cuda")
    par = torch.as_tensor(par_np, dtype=torch.int32, device="cuda")
    outs = B.VerifyOutputs(T)
    st = torch.cuda.current_stream()

    def step():
        B.oos_tree_verify(model, kv, ctx, tok, par, T, outs.accepted_len, outs.accepted_nodes, outs.accepted_tokens,
                          outs.bonus, st)

    for _ in range(3):
        step()
    torch.cuda.synchronize()
    assert L.oos_timeline_gemm_clear() == 0 and L.oos_timeline_attn_clear() == 0
    step()
    torch.cuda.synchronize()
    assert B.oos_last_status(model) == B.OOS_OK

    g = np.zeros((1024, 160, 6), np.uint64)
    assert L.oos_timeline_gemm_read(g.ctypes.data_as(ctypes.c_void_p), ctypes.c_size_t(g.nbytes)) == 0
    a = np.zeros((2048, 24), np.uint64)
    assert L.oos_timeline_attn_read(a.ctypes.data_as(ctypes.c_void_p), ctypes.c_size_t(a.nbytes)) == 0

    launches = []
    for i in range(g.shape[0]):
        b = g[i].astype(np.int64)
        b = b[b[:, 0] > 0]
        if len(b):
            launches.append((b[:, 0].min(), b))
    launches.sort(key=lambda x: x[0])
    t0 = launches[0][0]
    kinds = ["q/k/v", "O", "gate/up", "down"]
    agg = {k: [] for k in kinds}
    gaps = {k: [] for k in kinds}
    prev_exit = None
    for n, (start, b) in enumerate(launches):
        kind = kinds[n % 4]
        main_end = b[:, 2].max()
        publish = b[:, 4].max()
        pol = b[:, 5][b[:, 5] > 0]
        released = pol.max() if len(pol) else publish
        exit_ = b[:, 3].max()
        agg[kind].append(((main_end - start), (exit_ - main_end), (publish - main_end), (released - publish),
                          (exit_ - released)))
        if prev_exit is not None:
            gaps[kind].append(exit_ - prev_exit)
        prev_exit = exit_
    print("%s, T=%d, ctx_len=%d, %d layers: one graph-replayed step, %d GEMM launches"
          % (args.workload, T, ctx, cfg.n_layers, len(launches)))
    print("step: first GEMM entry -> last GEMM exit %.1f us" % ((launches[-1][1][:, 3].max() - t0) / 1e3))
    print("per GEMM kind, mean over layers (us):")
    for k in kinds:
        x = np.array(agg[k]) / 1e3
        gp = np.array(gaps[k]) / 1e3 if gaps[k] else np.zeros(1)
        print("  %-8s main %6.2f  tail %6.2f [publish %5.2f  poll %5.2f  finish %5.2f]  previous exit -> exit %6.2f"
              % (k, x[:, 0].mean(), x[:, 1].mean(), x[:, 2].mean(), x[:, 3].mean(), x[:, 4].mean(), gp.mean()))
    print("  (the O row's 'previous exit -> exit' includes the attention)")

    b = a.astype(np.int64)
    b = b[b[:, 0] > 0]
    if len(b):
        ta = b[:, 0].min()
        names = [(0, "entry"), (1, "dependency wait done"), (2, "q landed")]
        for t in range(6):
            names += [(3 + 2 * t, "softmax tile %d start" % t), (4 + 2 * t, "softmax tile %d end" % t)]
        names += [(15, "all MMAs done"), (21, "merge rows staged"), (22, "cluster barrier passed"),
                  (16, "rows copied out"), (17, "own rows received"), (18, "exit")]
        print("last attention launch: %d blocks, %d splits, %d-%d tiles per block (us from the first entry, "
              "median over blocks [max])" % (len(b), b[0, 20], b[:, 19].min(), b[:, 19].max()))
        for e, label in names:
            col = b[:, e]
            col = col[col > 0] - ta
            if len(col):
                print("  %-24s %7.2f [%7.2f]" % (label, np.median(col) / 1e3, col.max() / 1e3))
    model.close()


if __name__ == "__main__":
    main()
