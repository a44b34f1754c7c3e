"""Oracle for greedy tree verification -- TEST INFRASTRUCTURE ONLY.

Only the test suite, the smoke check and the benchmark's CPU-baseline leg may
import this module.  It is a plain, slow, fp64 CPU restatement of what the
target verifier computes, written from the paper's definitions, and shares no
code with the CUDA path.

What the paper fixes:
  * Target authority (Eq. 1): under greedy decoding the next committed token
    is argmax_v p_T(v | x, y_<t).  The argmax of p_T equals the argmax of the
    logits, so no softmax over the vocabulary is needed.
  * Verify and commit (Sec. "Target-Only Verification and Recovery"): the
    candidate tree is evaluated in one forward pass, the longest prefix
    allowed by the greedy rule is committed, at the first mismatch the target's
    own next token continues decoding, and only states on the accepted path
    enter the committed KV cache.
  * The ToolSpec loop (Sec. "Background"): the target commits the longest
    approved prefix of the candidate tree each round.

What the paper leaves open, and the reading taken here:
  * Node 0 is the root: the last committed token, whose K/V is not cached
    yet.  It is always accepted.  Nodes are numbered parents-first.
  * A tree node attends to the committed cache plus its own ancestors
    (itself included): one forward pass over a tree is therefore the same as
    causal decoding along every root-to-leaf path.
  * RoPE position of node i is ctx_len + depth(i) (rotate-half convention).
    Llama-3.1 targets turn their low-frequency pairs slower, by the frequency
    rescaling published with that model (rope_inv_freq); the paper runs
    Llama-3.1-8B and does not restate it.
  * K and V are stored in the cache's format before anything attends to them
    (bf16 for the bf16 models, binary16 for an FP16 cache): the tree's own K/V
    go through the cache too.
  * "Longest prefix" is the deepest accepted node, lowest node id on ties;
    argmax ties go to the lowest vocabulary id.
  * The decoder is a pre-norm Llama/Qwen block: RMSNorm, q/k/v projections
    (optional bias), optional per-head q/k RMSNorm (Qwen3), RoPE, grouped-
    query attention, output projection, RMSNorm, SwiGLU MLP.

Model protocol (duck-typed; the seeded input module provides one):
  m.cfg                  object with n_layers, hidden, n_q_heads, n_kv_heads,
                         head_dim, intermediate, vocab, rms_eps, rope_theta
                         (and, for rescaled rotary frequencies, rope_factor,
                         rope_low_freq_factor, rope_high_freq_factor,
                         rope_orig_max_pos)
  m.layer(l)             dict of fp64 arrays: attn_norm[H], w_q[nq*d,H],
                         w_k[nkv*d,H], w_v[nkv*d,H], b_q/b_k/b_v (or None),
                         q_norm/k_norm [d] (or None), w_o[H,nq*d], mlp_norm[H],
                         w_gate[I,H], w_up[I,H], w_down[H,I]
  m.embed_rows(ids)      [n,H] fp64 embedding rows
  m.final_norm()         [H]
  m.lm_head_blocks()     iterator of (first_row, W_block[rows,H]) over the vocab
KV cache: per layer arrays k[l], v[l] of shape [n_pos, nkv, d] (fp64).
"""

import numpy as np


class TreeError(ValueError):
    """The parent array is not a parents-first tree rooted at node 0."""


# ---------------------------------------------------------------- tree shape

def tree_structure(parent):
    """Depth of every node and its root-to-node path (ancestors, itself last).

    Rejects parent[0] != -1 and any parent[i] outside [0, i).
    """
    parent = [int(p) for p in parent]
    T = len(parent)
    if T < 1:
        raise TreeError("empty tree")
    if parent[0] != -1:
        raise TreeError("node 0 must be the root (parent -1)")
    depth = [0]
    path = [[0]]
    for i in range(1, T):
        p = parent[i]
        if not (0 <= p < i):
            raise TreeError("parent[%d]=%d is not an earlier node" % (i, p))
        depth.append(depth[p] + 1)
        path.append(path[p] + [i])
    return depth, path


# ---------------------------------------------------------------- decoder ops

def rms_norm(x, gain, eps):
    """x / sqrt(mean(x^2) + eps) * gain over the last axis."""
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * gain


def rope_scaling(cfg):
    """(factor, low_freq_factor, high_freq_factor, original_context) of a
    model whose rotary frequencies are rescaled (Llama 3.1), else None."""
    f = float(getattr(cfg, "rope_factor", 0.0) or 0.0)
    if f <= 1.0:
        return None
    return (f, float(cfg.rope_low_freq_factor), float(cfg.rope_high_freq_factor), float(cfg.rope_orig_max_pos))


def rope_inv_freq(d, theta, scaling=None):
    """Turning rates of the d/2 dimension pairs: theta^(-2m/d), optionally
    rescaled the Llama 3.1 way.

    With scaling = (factor, low, high, L): a pair whose wavelength 2 pi / f is
    shorter than L / high keeps its rate; one longer than L / low turns factor
    times slower; in between the rate blends the two, weighted by
    (L / wavelength - low) / (high - low) towards the unscaled rate.
    """
    half = d // 2
    inv_freq = theta ** (-2.0 * np.arange(half, dtype=np.float64) / d)
    if scaling is None:
        return inv_freq
    factor, low, high, L = scaling
    out = np.empty_like(inv_freq)
    for m, f in enumerate(inv_freq):
        wavelen = 2.0 * np.pi / f
        if wavelen < L / high:
            out[m] = f
        elif wavelen > L / low:
            out[m] = f / factor
        else:
            w = (L / wavelen - low) / (high - low)
            out[m] = (1.0 - w) * f / factor + w * f
    return out


def rope(x, pos, theta, scaling=None):
    """Rotate-half rotary embedding of vectors x[..., d] at one position.

    Dimension pairs (m, m + d/2) turn by the angle pos * inv_freq[m], with
    inv_freq from rope_inv_freq (theta^(-2m/d) unless the model rescales it).
    """
    d = x.shape[-1]
    half = d // 2
    inv_freq = rope_inv_freq(d, theta, scaling)
    ang = float(pos) * inv_freq
    c, s = np.cos(ang), np.sin(ang)
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


def silu(z):
    return z / (1.0 + np.exp(-z))


def cache_format(x, dtype):
    """K or V as the KV cache stores it.

    The target's KV cache is kept in the model's precision (the paper's targets
    run BF16 or FP16 caches): a bf16 cache stores round-to-nearest-even bf16
    values, so every K/V a node attends to -- cached or written by the tree
    pass itself -- is bf16.  An fp16 cache (the paper's Qwen2.5 and Llama
    backend) stores the fp32 value rounded to IEEE binary16, nearest-even,
    overflowing to infinity.  An fp32 cache is kept exact here (fp32 rounding
    of K/V is far below the fp32 tolerance).
    """
    if dtype == "f16":
        with np.errstate(over="ignore"):          # overflow to infinity is the format's rule
            return np.asarray(x, dtype=np.float32).astype(np.float16).astype(np.float64)
    if dtype != "bf16":
        return x
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return (u.astype(np.uint32) << 16).view(np.float32).astype(np.float64).reshape(np.shape(x))


def kv_format(cfg):
    """Element type of the model's KV cache: cfg.cache_dtype when set (the
    FP16 cache backend of the paper's Qwen2.5 and Llama runs, "Targets,
    Workloads, and Protocol"), else the model dtype."""
    return getattr(cfg, "cache_dtype", "") or cfg.dtype


def attend(q, keys, values):
    """softmax(keys q / sqrt(d)) @ values for one query vector."""
    d = q.shape[-1]
    s = keys @ q / np.sqrt(d)
    s = s - s.max()
    p = np.exp(s)
    p = p / p.sum()
    return p @ values


def qkv(W, cfg, h):
    """q [n,nq,d], k [n,nkv,d], v [n,nkv,d] of normalised inputs h [n,H]."""
    n = h.shape[0]
    d = cfg.head_dim
    q = h @ W["w_q"].T
    k = h @ W["w_k"].T
    v = h @ W["w_v"].T
    if W.get("b_q") is not None:
        q = q + W["b_q"]
        k = k + W["b_k"]
        v = v + W["b_v"]
    q = q.reshape(n, cfg.n_q_heads, d)
    k = k.reshape(n, cfg.n_kv_heads, d)
    v = v.reshape(n, cfg.n_kv_heads, d)
    if W.get("q_norm") is not None:
        q = rms_norm(q, W["q_norm"], cfg.rms_eps)
        k = rms_norm(k, W["k_norm"], cfg.rms_eps)
    return q, k, v


def mlp(W, cfg, x):
    h = rms_norm(x, W["mlp_norm"], cfg.rms_eps)
    return (silu(h @ W["w_gate"].T) * (h @ W["w_up"].T)) @ W["w_down"].T


def lm_head_argmax(m, hf):
    """Greedy token of each row of hf (Eq. 1), with the top-1 and top-2 logits.

    Ties go to the lowest vocabulary id; top2 is the second largest logit
    counted with multiplicity (equal to top1 when the maximum is repeated).
    """
    n = hf.shape[0]
    best = np.full(n, -np.inf)
    arg = np.zeros(n, np.int64)
    second = np.full(n, -np.inf)
    for r0, Wb in m.lm_head_blocks():
        logits = hf @ Wb.T                       # [n, rows]
        for i in range(n):
            row = logits[i]
            j = int(np.argmax(row))              # first maximum of the block
            v = row[j]
            rest = np.delete(row, j)
            v2 = rest.max() if rest.size else -np.inf
            if v > best[i]:
                second[i] = max(best[i], v2)
                best[i], arg[i] = v, r0 + j
            else:
                second[i] = max(second[i], v)    # v <= best: v is a runner-up
    return arg, best, second


# ---------------------------------------------------------------- tree pass

def verify_tree(m, cache_k, cache_v, ctx_len, tokens, parent, only=None):
    """One forward pass of the target over a candidate tree.

    Node i sees the ctx_len committed positions and its own ancestors, at RoPE
    position ctx_len + depth(i).  Returns a dict with
      final_hidden [T,H] (output of the final RMSNorm), argmax/top1/top2 [T],
      tree_k / tree_v: per layer [T,nkv,d] (post-RoPE K and V of every node),
    Rows of nodes outside `only` (and its ancestor closure) are left NaN.
    """
    cfg = m.cfg
    depth, path = tree_structure(parent)
    T = len(tokens)
    nodes = list(range(T))
    if only is not None:
        keep = set()
        for i in only:
            keep.update(path[i])
        nodes = sorted(keep)
    nq, nkv, d = cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim
    group = nq // nkv
    x = np.full((T, cfg.hidden), np.nan)
    x[nodes] = m.embed_rows(np.asarray(tokens)[nodes])
    tree_k, tree_v = [], []
    for l in range(cfg.n_layers):
        W = m.layer(l)
        h = rms_norm(x[nodes], W["attn_norm"], cfg.rms_eps)
        q_s, k_s, v_s = qkv(W, cfg, h)
        q = np.full((T, nq, d), np.nan)
        k = np.full((T, nkv, d), np.nan)
        v = np.full((T, nkv, d), np.nan)
        for r, i in enumerate(nodes):
            q[i] = rope(q_s[r], ctx_len + depth[i], cfg.rope_theta, rope_scaling(cfg))
            k[i] = cache_format(rope(k_s[r], ctx_len + depth[i], cfg.rope_theta, rope_scaling(cfg)), kv_format(cfg))
            v[i] = cache_format(v_s[r], kv_format(cfg))
        tree_k.append(k)
        tree_v.append(v)
        o = np.zeros((T, nq, d))
        for i in nodes:
            for hd in range(nq):
                g = hd // group
                keys = np.concatenate([cache_k[l][:ctx_len, g], k[path[i], g]])
                vals = np.concatenate([cache_v[l][:ctx_len, g], v[path[i], g]])
                o[i, hd] = attend(q[i, hd], keys, vals)
        x[nodes] = x[nodes] + o[nodes].reshape(len(nodes), nq * d) @ W["w_o"].T
        x[nodes] = x[nodes] + mlp(W, cfg, x[nodes])
    hf = np.full((T, cfg.hidden), np.nan)
    hf[nodes] = rms_norm(x[nodes], m.final_norm(), cfg.rms_eps)
    argmax = np.full(T, -1, np.int64)
    top1 = np.full(T, np.nan)
    top2 = np.full(T, np.nan)
    a, t1, t2 = lm_head_argmax(m, hf[nodes])
    argmax[nodes], top1[nodes], top2[nodes] = a, t1, t2
    return dict(final_hidden=hf, argmax=argmax, top1=top1, top2=top2,
                tree_k=tree_k, tree_v=tree_v, depth=np.asarray(depth), nodes=nodes)


# ---------------------------------------------------------------- accept / commit

def accept(tokens, parent, argmax):
    """Greedy longest-prefix acceptance over the tree.

    The root is accepted; a draft node is accepted when its parent is and its
    token equals the target's greedy choice at the parent.  The committed path
    runs from the root to the deepest accepted node (lowest id among equally
    deep ones); the bonus token is the target's own choice after that node.
    """
    depth, path = tree_structure(parent)
    T = len(tokens)
    ok = [False] * T
    ok[0] = True
    for i in range(1, T):
        p = int(parent[i])
        ok[i] = ok[p] and int(tokens[i]) == int(argmax[p])
    deepest = 0
    for i in range(T):
        if ok[i] and depth[i] > depth[deepest]:
            deepest = i
    nodes = path[deepest]
    return dict(accepted_len=len(nodes), accepted_nodes=list(nodes),
                accepted_tokens=[int(tokens[i]) for i in nodes],
                bonus=int(argmax[deepest]))


def compact(cache_k, cache_v, ctx_len, accepted_nodes):
    """Move the accepted path's K/V into the committed slots.

    Slot ctx_len + j receives the entry that tree node accepted_nodes[j] wrote
    to slot ctx_len + accepted_nodes[j], read from the cache as it was before
    the move (a gather from a snapshot).  Arrays are [capacity, nkv, d] per
    layer and are returned as new arrays.
    """
    out_k, out_v = [], []
    for ck, cv in zip(cache_k, cache_v):
        snap_k, snap_v = ck.copy(), cv.copy()
        nk, nv = ck.copy(), cv.copy()
        for j, src in enumerate(accepted_nodes):
            nk[ctx_len + j] = snap_k[ctx_len + src]
            nv[ctx_len + j] = snap_v[ctx_len + src]
        out_k.append(nk)
        out_v.append(nv)
    return out_k, out_v


def verify_and_accept(m, cache_k, cache_v, ctx_len, tokens, parent):
    r = verify_tree(m, cache_k, cache_v, ctx_len, tokens, parent)
    r.update(accept(tokens, parent, r["argmax"]))
    return r


# ---------------------------------------------------------------- plain decoding

def decode_step(m, cache_k, cache_v, n_pos, token):
    """Ordinary causal decoding of one token at position n_pos.

    Attends to cache positions 0..n_pos-1 and to itself; returns
    (final_hidden[H], argmax, top1, top2, k_per_layer, v_per_layer).
    The caller appends the returned K/V to the cache.
    """
    cfg = m.cfg
    nq, nkv, d = cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim
    group = nq // nkv
    x = m.embed_rows([token])                  # [1, H]
    ks, vs = [], []
    for l in range(cfg.n_layers):
        W = m.layer(l)
        h = rms_norm(x, W["attn_norm"], cfg.rms_eps)
        q, k, v = qkv(W, cfg, h)
        q = rope(q[0], n_pos, cfg.rope_theta, rope_scaling(cfg))
        k = cache_format(rope(k[0], n_pos, cfg.rope_theta, rope_scaling(cfg)), kv_format(cfg))
        v = cache_format(v[0], kv_format(cfg))
        ks.append(k)
        vs.append(v)
        o = np.zeros((nq, d))
        for hd in range(nq):
            g = hd // group
            keys = np.concatenate([cache_k[l][:n_pos, g], k[g][None]])
            vals = np.concatenate([cache_v[l][:n_pos, g], v[g][None]])
            o[hd] = attend(q[hd], keys, vals)
        x = x + o.reshape(1, nq * d) @ W["w_o"].T
        x = x + mlp(W, cfg, x)
    hf = rms_norm(x, m.final_norm(), cfg.rms_eps)
    a, t1, t2 = lm_head_argmax(m, hf)
    return hf[0], int(a[0]), float(t1[0]), float(t2[0]), ks, vs


def decode_sequence(m, cache_k, cache_v, n_pos, tokens):
    """Causal decoding of a token sequence after n_pos cached positions.

    Returns per-step outputs and the extended caches (new arrays).
    """
    ck = [np.array(c[:n_pos]) for c in cache_k]
    cv = [np.array(c[:n_pos]) for c in cache_v]
    steps = []
    for t in tokens:
        hf, a, t1, t2, ks, vs = decode_step(m, ck, cv, n_pos, int(t))
        ck = [np.concatenate([c, k[None]]) for c, k in zip(ck, ks)]
        cv = [np.concatenate([c, v[None]]) for c, v in zip(cv, vs)]
        n_pos += 1
        steps.append(dict(final_hidden=hf, argmax=a, top1=t1, top2=t2, k=ks, v=vs))
    return steps, ck, cv


def prefill(m, tokens):
    """K/V cache of a prompt by causal decoding from an empty cache."""
    cfg = m.cfg
    empty = [np.zeros((0, cfg.n_kv_heads, cfg.head_dim)) for _ in range(cfg.n_layers)]
    steps, ck, cv = decode_sequence(m, empty, empty, 0, tokens)
    return ck, cv, steps


def greedy_continuation(m, cache_k, cache_v, n_pos, root, n):
    """The target's own next n tokens after `root` (Eq. 1 applied n times),
    with the top-1/top-2 margin of each decision."""
    ck = [np.array(c[:n_pos]) for c in cache_k]
    cv = [np.array(c[:n_pos]) for c in cache_v]
    out, margins = [], []
    tok = int(root)
    for _ in range(n):
        hf, a, t1, t2, ks, vs = decode_step(m, ck, cv, n_pos, tok)
        ck = [np.concatenate([c, k[None]]) for c, k in zip(ck, ks)]
        cv = [np.concatenate([c, v[None]]) for c, v in zip(cv, vs)]
        n_pos += 1
        out.append(a)
        margins.append(t1 - t2)
        tok = a
    return out, margins
