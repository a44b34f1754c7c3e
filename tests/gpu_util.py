"""Helpers of the GPU parity tests: run the CUDA path through the C ABI and
compare it with the CPU checker on the same seeded inputs."""

import numpy as np
import torch

import oracle
from paper_2608_00814_gb300 import binding as B
from synth.device import upload_cache, upload_model

# Tolerances.  bf16 configs: the bound the method's own precision allows
# (max-abs error <= 2e-2 * max(1, max|oracle|) per tensor; bit-exact accept
# outputs where every accepted node's top-1/top-2 logit margin exceeds 0.05).
# fp32 configs: fp32 accumulation over K <= 512 terms keeps errors near 1e-6
# relative, so 1e-4 and a 1e-4 margin gate leave two orders of headroom.
TOL = {"bf16": 2e-2, "f32": 1e-4}
GATE = {"bf16": 0.05, "f32": 1e-4}


def gpu_model(case, max_T=128, use_graph=True):
    w = upload_model(case.model)
    return B.OosModel(case.cfg, w, max_T=max_T, use_graph=use_graph), w


def gpu_cache(case, capacity):
    k, v = upload_cache(case.cfg, case.cache_native, capacity)
    return B.KVCache(k, v)


def to_f64(cfg, t):
    return t.detach().float().cpu().numpy().astype(np.float64)


def _bits(t):
    return t.view(torch.int16) if t.element_size() == 2 else t.view(torch.int32)


def run(model, kv, ctx, tokens, parent, outs=None):
    """One tree through both verify entry points on the same cache: first
    oos_tree_verify (the call the benchmark times), then
    oos_tree_verify_debug (the same step plus final hidden rows and per-node
    argmax / top-1 / top-2).  The two must agree bit for bit on the accept
    outputs and on the tree K/V they write; the debug call's intermediates
    are returned for the comparison with the CPU checker, and the plain call's
    accept outputs feed the compaction check.  `outs`, when given, is a pair of
    output buffer sets (plain, debug) reused from call to call."""
    tok = torch.as_tensor(np.asarray(tokens, np.int32), device="cuda")
    par = torch.as_tensor(np.asarray(parent, np.int32), device="cuda")
    T = len(tokens)
    plain = B.tree_verify(model, kv, ctx, tok, par, outs=outs[0] if outs else None, debug=False)
    torch.cuda.synchronize()
    plain_status = B.oos_last_status(model)
    plain_k = [_bits(kv.k[l][ctx:ctx + T]).clone() for l in range(len(kv.k))]
    plain_v = [_bits(kv.v[l][ctx:ctx + T]).clone() for l in range(len(kv.v))]
    outs = B.tree_verify(model, kv, ctx, tok, par, outs=outs[1] if outs else None, debug=True)
    torch.cuda.synchronize()
    status = B.oos_last_status(model)
    assert status == plain_status, (status, plain_status)
    n = int(outs.accepted_len.item())
    for a, b in ((plain.accepted_len, outs.accepted_len), (plain.accepted_nodes, outs.accepted_nodes),
                 (plain.accepted_tokens, outs.accepted_tokens), (plain.bonus, outs.bonus)):
        assert torch.equal(a, b), "oos_tree_verify and oos_tree_verify_debug disagree"
    for l in range(len(kv.k)):
        assert torch.equal(plain_k[l], _bits(kv.k[l][ctx:ctx + T])) and \
            torch.equal(plain_v[l], _bits(kv.v[l][ctx:ctx + T])), "tree K/V differ between the entry points"
    return dict(status=status, accepted_len=n,
                accepted_nodes=outs.accepted_nodes.cpu().numpy().tolist(),
                accepted_tokens=outs.accepted_tokens.cpu().numpy().tolist(),
                bonus=int(outs.bonus.item()), final_hidden=outs.final_hidden.cpu().numpy().astype(np.float64),
                argmax=outs.argmax.cpu().numpy(), top1=outs.top1.cpu().numpy(), top2=outs.top2.cpu().numpy(),
                tree_k=[to_f64(None, kv.k[l][ctx:ctx + T]) for l in range(len(kv.k))],
                tree_v=[to_f64(None, kv.v[l][ctx:ctx + T]) for l in range(len(kv.v))],
                plain=dict(accepted_len=int(plain.accepted_len.item()),
                           accepted_nodes=plain.accepted_nodes.cpu().numpy().tolist(),
                           accepted_tokens=plain.accepted_tokens.cpu().numpy().tolist(),
                           bonus=int(plain.bonus.item())),
                outs=plain, debug_outs=outs, tok=tok, par=par)


def max_rel_err(gpu, ref, rows=None):
    if rows is not None:
        gpu, ref = gpu[rows], ref[rows]
    scale = max(1.0, float(np.abs(ref).max()))
    return float(np.abs(gpu - ref).max()) / scale


def ok_nodes(tokens, parent, argmax):
    T = len(tokens)
    ok = [False] * T
    ok[0] = True
    for i in range(1, T):
        ok[i] = ok[parent[i]] and int(tokens[i]) == int(argmax[parent[i]])
    return [i for i in range(T) if ok[i]]


def check_case(case, g, r, rows=None, tol=None, gate=None):
    """Compare a GPU result g with the oracle result r.  Returns True when the
    case passed the margin gate (accept outputs compared exactly)."""
    dt = case.cfg.dtype
    tol = TOL[dt] if tol is None else tol
    gate = GATE[dt] if gate is None else gate
    rows = list(range(len(case.tokens))) if rows is None else rows
    assert g["status"] == B.OOS_OK
    e = max_rel_err(g["final_hidden"], r["final_hidden"], rows)
    assert e <= tol, "final hidden error %.3g > %.3g" % (e, tol)
    for l in range(case.cfg.n_layers):
        ek = max_rel_err(g["tree_k"][l], r["tree_k"][l], rows)
        ev = max_rel_err(g["tree_v"][l], r["tree_v"][l], rows)
        assert ek <= tol and ev <= tol, "layer %d tree K/V error %.3g/%.3g" % (l, ek, ev)
    # the largest and second-largest logit of every node, same tolerance
    for key in ("top1", "top2"):
        e = max_rel_err(g[key].astype(np.float64), r[key], rows)
        assert e <= tol, "%s logit error %.3g > %.3g" % (key, e, tol)
    margin = r["top1"] - r["top2"]
    for i in rows:
        if margin[i] > gate:
            assert g["argmax"][i] == r["argmax"][i], (i, g["argmax"][i], r["argmax"][i], margin[i])
    okn = ok_nodes(case.tokens, case.parent, r["argmax"])
    gated = all(margin[i] > gate for i in okn)
    if gated:
        a = oracle.accept(case.tokens, case.parent, r["argmax"])
        for out in (g, g["plain"]):    # the debug call and the timed call
            assert out["accepted_len"] == a["accepted_len"]
            assert out["accepted_nodes"][:a["accepted_len"]] == a["accepted_nodes"]
            assert out["accepted_tokens"][:a["accepted_len"]] == a["accepted_tokens"]
            assert all(x == -1 for x in out["accepted_nodes"][a["accepted_len"]:])
            assert all(x == -1 for x in out["accepted_tokens"][a["accepted_len"]:])
            assert out["bonus"] == a["bonus"]
    return gated


def check_compaction(model, kv, ctx, g):
    """GPU compaction == gather from a snapshot, bit for bit, on every layer.
    The accept outputs compacted are those of oos_tree_verify (the timed
    entry point), as the benchmark step uses them."""
    T = len(g["accepted_nodes"])
    snap_k = [t.clone() for t in kv.k]
    snap_v = [t.clone() for t in kv.v]
    B.oos_kv_compact(model, kv, ctx, g["outs"].accepted_nodes, g["outs"].accepted_len, T)
    torch.cuda.synchronize()
    n = g["accepted_len"]
    path = g["accepted_nodes"][:n]
    for l in range(len(kv.k)):
        for snap, cur in ((snap_k[l], kv.k[l]), (snap_v[l], kv.v[l])):
            exp = snap.clone()
            for j, src in enumerate(path):
                exp[ctx + j] = snap[ctx + src]
            assert torch.equal(_bits(exp), _bits(cur))
