// Small kernels of the verify step: tree preparation, embedding, the GEMM
// reduce-epilogues (q/k/v with RoPE, residual + RMSNorm, SwiGLU), the argmax
// merge with the greedy-acceptance walk, and KV compaction.
#include <math.h>

#include <vector>

#include "common.cuh"
#include "internal.h"

namespace oos {

// ============================================================ tree preparation
// Tree encoding: parents-first numbering (parent[0] = -1, parent[i] < i).  Node
// i attends to the committed cache and its ancestors (itself included); its
// RoPE position is ctx + depth(i).  Ancestor sets are 128-bit masks.
// ctx: the committed length, from the host (ctx_in == nullptr) or from device
// memory; written to ctx_out, where every later kernel of the step reads it.
__global__ void __launch_bounds__(kMaxT) k_tree_prep(const int32_t* __restrict__ tokens,
                                                     const int32_t* __restrict__ parent, int T, int ctx,
                                                     const int32_t* __restrict__ ctx_in, int32_t* ctx_out,
                                                     int vocab, uint32_t* status, int32_t* depth_out,
                                                     int32_t* pos_out, unsigned long long* anc_out) {
  __shared__ int s_parent[kMaxT];
  __shared__ int s_bad;
  pdl_wait();
  pdl_trigger();
  if (ctx_in) ctx = *ctx_in;
  const int i = threadIdx.x;
  if (i == 0) *ctx_out = ctx;
  if (i == 0) s_bad = 0;
  __syncthreads();
  if (i < T) {
    const int p = parent[i];
    const int tok = tokens[i];
    const bool ok = (i == 0 ? p == -1 : (p >= 0 && p < i)) && tok >= 0 && tok < vocab;
    s_parent[i] = p;
    if (!ok) atomicOr(&s_bad, 1);
  }
  __syncthreads();
  if (i == 0) *status = s_bad ? ST_TREE : 0u;
  if (i >= 1 && i < 8) status[i] = 0u;   // where a pipeline wait gave up (see common.cuh)
  if (i < T) {
    int d = 0;
    unsigned long long lo = 0, hi = 0;
    if (!s_bad) {
      for (int a = i; a >= 0; a = (a == 0 ? -1 : s_parent[a])) {
        if (a < 64) lo |= 1ull << a; else hi |= 1ull << (a - 64);
        if (a != i) ++d;
      }
    } else {
      if (i < 64) lo = 1ull << i; else hi = 1ull << (i - 64);
    }
    depth_out[i] = d;
    pos_out[i] = ctx + d;
    anc_out[2 * i] = lo;
    anc_out[2 * i + 1] = hi;
  }
}

// The first kernel of a step is launched without programmatic serialisation:
// it starts only after all earlier work on the stream (the previous step's
// compaction, the caller's cache writes) has completed.  Every kernel of the
// step lets its dependents launch only after its own dependency wait, so a
// kernel that starts finds the kernel two launches back, and all before it,
// complete: later kernels may read cache positions < ctx, and ctx itself,
// before their own dependency wait.
cudaError_t launch_tree_prep(Model& m, const int32_t* tokens, const int32_t* parent, int T, int ctx,
                             const int32_t* ctx_dev, cudaStream_t st) {
  return launch(false, k_tree_prep, dim3(1), dim3(kMaxT), 0, st, tokens, parent, T, ctx, ctx_dev, m.ws.ctx,
                m.cfg.vocab, m.ws.status, m.ws.depth, m.ws.pos, m.ws.anc);
}

cudaGraphNode_t find_tree_prep_node(cudaGraph_t g) {
  size_t n = 0;
  if (cudaGraphGetNodes(g, nullptr, &n) != cudaSuccess || n == 0) return nullptr;
  std::vector<cudaGraphNode_t> nodes(n);
  if (cudaGraphGetNodes(g, nodes.data(), &n) != cudaSuccess) return nullptr;
  for (size_t i = 0; i < n; ++i) {
    cudaGraphNodeType t;
    if (cudaGraphNodeGetType(nodes[i], &t) != cudaSuccess || t != cudaGraphNodeTypeKernel) continue;
    cudaKernelNodeParams p;
    if (cudaGraphKernelNodeGetParams(nodes[i], &p) != cudaSuccess) continue;
    if (p.func == (void*)k_tree_prep) return nodes[i];
  }
  return nullptr;
}

// the same arguments launch_tree_prep passes, with another committed length
cudaError_t set_tree_prep_ctx(Model& m, cudaGraphExec_t ex, cudaGraphNode_t node, const int32_t* tokens,
                              const int32_t* parent, int T, int ctx) {
  const int32_t* ctx_in = nullptr;
  int32_t* ctx_out = m.ws.ctx;
  int vocab = m.cfg.vocab;
  uint32_t* status = m.ws.status;
  int32_t* depth = m.ws.depth;
  int32_t* pos = m.ws.pos;
  unsigned long long* anc = m.ws.anc;
  void* args[] = {&tokens, &parent, &T, &ctx, &ctx_in, &ctx_out, &vocab, &status, &depth, &pos, &anc};
  cudaKernelNodeParams p = {};
  p.func = (void*)k_tree_prep;
  p.gridDim = dim3(1);
  p.blockDim = dim3(kMaxT);
  p.sharedMemBytes = 0;
  p.kernelParams = args;
  return cudaGraphExecKernelNodeSetParams(ex, node, &p);
}

// ============================================================ embedding + first RMSNorm
// x[t] = E[token_t] (fp32 residual); xn[t] = x * rsqrt(mean(x^2) + eps) * g.
template <typename E>
__global__ void __launch_bounds__(256) k_embed_norm(const int32_t* __restrict__ tokens, const E* __restrict__ emb,
                                                    const E* __restrict__ gain, int H, int vocab, float eps,
                                                    float* __restrict__ x, E* __restrict__ xn) {
  __shared__ float red[32];
  pdl_wait();
  pdl_trigger();
  const int t = blockIdx.x;
  int tok = tokens[t];
  tok = tok < 0 ? 0 : (tok >= vocab ? vocab - 1 : tok);   // invalid trees are flagged by tree_prep
  const E* row = emb + (size_t)tok * H;
  float ss = 0.f;
  for (int f = threadIdx.x; f < H; f += blockDim.x) {
    const float v = to_f32(row[f]);
    x[(size_t)t * H + f] = v;
    ss += v * v;
  }
  ss = block_sum(ss, red);
  const float r = rsqrtf(ss / (float)H + eps);
  for (int f = threadIdx.x; f < H; f += blockDim.x)
    store_act(xn, (size_t)t * H + f, (size_t)kMaxT * H, x[(size_t)t * H + f] * r * to_f32(gain[f]));
}

cudaError_t launch_embed_norm(Model& m, const int32_t* tokens, int T, cudaStream_t st) {
  const auto& c = m.cfg;
  if (c.dtype == OOS_DTYPE_BF16)
    return launch(m.pdl, k_embed_norm<__nv_bfloat16>, dim3(T), dim3(256), 0, st, tokens,
                  (const __nv_bfloat16*)m.w.embed, (const __nv_bfloat16*)m.layers[0].attn_norm, c.hidden,
                  c.vocab, c.rms_eps, m.ws.x, (__nv_bfloat16*)m.ws.xn);
  return launch(m.pdl, k_embed_norm<float>, dim3(T), dim3(256), 0, st, tokens, (const float*)m.w.embed,
                (const float*)m.layers[0].attn_norm, c.hidden, c.vocab, c.rms_eps, m.ws.x, (float*)m.ws.xn);
}

// bf16 path: the first RMSNorm is folded into the QKV GEMM.  Block (t, chunk)
// writes x = E[token] (fp32 residual), y = g (.) x (hi/lo bf16 GEMM input) and
// the chunk's sum of x^2 (the GEMM epilogue turns the chunk sums into
// rsqrt(mean(x^2) + eps)).
// Block (t, 0) also fills the step's RoPE table: cos/sin of pos[t] * theta^(-2m/d)
// for m < d/2, the angle formed and reduced to [-pi, pi] in fp64 once per step
// (every layer reuses it).
__global__ void __launch_bounds__(128) k_embed_tc(const int32_t* __restrict__ tokens, const __nv_bfloat16* __restrict__ emb,
                                                  const __nv_bfloat16* __restrict__ gain, int H, int vocab,
                                                  float* __restrict__ x, __nv_bfloat16* __restrict__ y,
                                                  float* __restrict__ ss, const int32_t* __restrict__ pos,
                                                  const double* __restrict__ inv_freq, int half_d,
                                                  float2* __restrict__ rope, int* __restrict__ cnt, int n_cnt) {
  __shared__ float red[32];
  pdl_wait();
  pdl_trigger();
  const int t = blockIdx.x, f = blockIdx.y * 128 + threadIdx.x;
  {   // the step's GEMM arrival counters start from zero
    const int nb = gridDim.x * gridDim.y, b = blockIdx.y * gridDim.x + blockIdx.x;
    for (int i = b * blockDim.x + threadIdx.x; i < n_cnt; i += nb * blockDim.x) cnt[i] = 0;
  }
  if (blockIdx.y == 0 && threadIdx.x < half_d) {
    const double two_pi = 6.283185307179586476925286766559;
    const double ang = (double)pos[t] * inv_freq[threadIdx.x];
    float sn, cs;
    sincosf((float)(ang - two_pi * rint(ang / two_pi)), &sn, &cs);
    rope[t * half_d + threadIdx.x] = make_float2(cs, sn);
  }
  int tok = tokens[t];
  tok = tok < 0 ? 0 : (tok >= vocab ? vocab - 1 : tok);   // invalid trees are flagged by tree_prep
  float v = 0.f;
  if (f < H) {
    v = __bfloat162float(emb[(size_t)tok * H + f]);
    x[(size_t)t * H + f] = v;
    store_act(y, (size_t)t * H + f, (size_t)kMaxT * H, v * __bfloat162float(gain[f]));
  }
  const float s = block_sum(v * v, red);
  if (threadIdx.x == 0) ss[(size_t)blockIdx.y * kMaxT + t] = s;
}

cudaError_t launch_embed_tc(Model& m, const int32_t* tokens, int T, cudaStream_t st) {
  const auto& c = m.cfg;
  return launch(m.pdl, k_embed_tc, dim3(T, (c.hidden + 127) / 128), dim3(128), 0, st, tokens,
                (const __nv_bfloat16*)m.w.embed, (const __nv_bfloat16*)m.layers[0].attn_norm, c.hidden, c.vocab,
                m.ws.x, (__nv_bfloat16*)m.ws.xn, m.ws.ss, (const int32_t*)m.ws.pos, (const double*)m.ws.inv_freq,
                c.head_dim / 2, m.ws.rope, m.ws.cnt, c.n_layers * 4 * kCntPer);
}

// bf16 path, checking output only: the final RMSNorm output in fp32,
// hidden[t] = x[t] * rsqrt(mean(x[t]^2) + eps) * g.
__global__ void __launch_bounds__(256) k_final_hidden(const float* __restrict__ x, const float* __restrict__ ss,
                                                      int chunks, const __nv_bfloat16* __restrict__ gain, int H,
                                                      float eps, float* __restrict__ hidden) {
  pdl_wait();
  pdl_trigger();
  const int t = blockIdx.x;
  float s = 0.f;
  for (int c = 0; c < chunks; ++c) s += ss[(size_t)c * kMaxT + t];
  const float r = rsqrtf(s / (float)H + eps);
  for (int f = threadIdx.x; f < H; f += blockDim.x)
    hidden[(size_t)t * H + f] = x[(size_t)t * H + f] * r * __bfloat162float(gain[f]);
}

cudaError_t launch_final_hidden(Model& m, float* hidden, int T, cudaStream_t st) {
  const auto& c = m.cfg;
  return launch(m.pdl, k_final_hidden, dim3(T), dim3(256), 0, st, (const float*)m.ws.x, (const float*)m.ws.ss,
                (c.hidden + 127) / 128, (const __nv_bfloat16*)m.w.final_norm, c.hidden, c.rms_eps, hidden);
}

// sum of the fp32 partial slices of GEMM output (t, f)
OOS_DEV float gather_partial(const float* __restrict__ part, const StreamK& plan, int N, int t, int f) {
  int c0, c1;
  plan.contributors(f / kTile, c0, c1);
  float v = 0.f;
  const size_t slice = (size_t)kMaxT * N;
  for (int s = 0; s <= c1 - c0; ++s) v += part[s * slice + (size_t)t * N + f];
  return v;
}

// ============================================================ q/k/v epilogue
// One block per (node t, head slot hs in [0, nq + 2 nkv)); thread j owns the
// rotate-half pair (j, j + d/2).  q/k: optional per-head RMSNorm, then RoPE at
// pos[t]; q goes to the query buffer, k and v to cache slot ctx + t.
struct QkvPostArgs {
  const float* part;
  StreamK plan;
  int N, nq, nkv, d;
  const void* bq;
  const void* bk;
  const void* bv;
  const void* gq;
  const void* gk;
  float eps;
  const int32_t* pos;
  const double* inv_freq;
  void* q;
  void* kc;
  void* vc;
  const int32_t* ctx;   // committed length of the step (device)
};

template <typename E>
__global__ void k_qkv_post(QkvPostArgs a) {
  __shared__ float red[32];
  pdl_wait();
  pdl_trigger();
  const int t = blockIdx.x, hs = blockIdx.y, j = threadIdx.x, half = a.d / 2;
  const int f0 = hs * a.d + j, f1 = f0 + half;
  float v0 = gather_partial(a.part, a.plan, a.N, t, f0);
  float v1 = gather_partial(a.part, a.plan, a.N, t, f1);
  int kind, h;  // 0 = q, 1 = k, 2 = v
  if (hs < a.nq) { kind = 0; h = hs; }
  else if (hs < a.nq + a.nkv) { kind = 1; h = hs - a.nq; }
  else { kind = 2; h = hs - a.nq - a.nkv; }
  const E* bias = (const E*)(kind == 0 ? a.bq : kind == 1 ? a.bk : a.bv);
  if (bias) {
    v0 += to_f32(bias[h * a.d + j]);
    v1 += to_f32(bias[h * a.d + j + half]);
  }
  if (kind < 2) {
    const E* g = (const E*)(kind == 0 ? a.gq : a.gk);
    if (g) {
      const float ss = block_sum(v0 * v0 + v1 * v1, red);
      const float r = rsqrtf(ss / (float)a.d + a.eps);
      v0 = v0 * r * to_f32(g[j]);
      v1 = v1 * r * to_f32(g[j + half]);
    }
    // angle = pos * theta^(-2j/d), reduced to [-pi, pi] before the fp32 sincos
    const double ang = (double)a.pos[t] * a.inv_freq[j];
    const double two_pi = 6.283185307179586476925286766559;
    const float red_ang = (float)(ang - two_pi * rint(ang / two_pi));
    float s, c;
    sincosf(red_ang, &s, &c);
    const float o0 = v0 * c - v1 * s;
    const float o1 = v1 * c + v0 * s;
    v0 = o0;
    v1 = o1;
  }
  E* dst;
  if (kind == 0) dst = (E*)a.q + ((size_t)t * a.nq + h) * a.d;
  else dst = (E*)(kind == 1 ? a.kc : a.vc) + ((size_t)(*a.ctx + t) * a.nkv + h) * a.d;
  dst[j] = from_f32<E>(v0);
  dst[j + half] = from_f32<E>(v1);
}

cudaError_t launch_qkv_post(Model& m, int layer, const StreamK& plan, void* kc, void* vc, int T, cudaStream_t st) {
  const auto& c = m.cfg;
  const auto& L = m.layers[layer];
  QkvPostArgs a;
  a.part = m.ws.part;
  a.plan = plan;
  a.nq = c.n_q_heads;
  a.nkv = c.n_kv_heads;
  a.d = c.head_dim;
  a.N = (c.n_q_heads + 2 * c.n_kv_heads) * c.head_dim;
  a.bq = c.qkv_bias ? L.b_q : nullptr;
  a.bk = c.qkv_bias ? L.b_k : nullptr;
  a.bv = c.qkv_bias ? L.b_v : nullptr;
  a.gq = c.qk_norm ? L.q_norm : nullptr;
  a.gk = c.qk_norm ? L.k_norm : nullptr;
  a.eps = c.rms_eps;
  a.pos = m.ws.pos;
  a.inv_freq = m.ws.inv_freq;
  a.q = m.ws.q;
  a.kc = kc;
  a.vc = vc;
  a.ctx = m.ws.ctx;
  dim3 grid(T, c.n_q_heads + 2 * c.n_kv_heads);
  if (c.dtype == OOS_DTYPE_BF16) return launch(m.pdl, k_qkv_post<__nv_bfloat16>, grid, dim3(c.head_dim / 2), 0, st, a);
  return launch(m.pdl, k_qkv_post<float>, grid, dim3(c.head_dim / 2), 0, st, a);
}

// ============================================================ residual add + RMSNorm
// x[t] += sum of partial slices (O-projection or down-projection output);
// xn[t] = RMSNorm(x[t]) * gain (input of the next GEMM).  For the final norm
// the fp32 normalised row is also written to hidden_out (when given).
template <typename E>
__global__ void __launch_bounds__(256) k_resid_norm(const float* __restrict__ part, StreamK plan, int H,
                                                    const E* __restrict__ gain, float eps, float* __restrict__ x,
                                                    E* __restrict__ xn, float* __restrict__ hidden_out) {
  __shared__ float red[32];
  pdl_wait();
  pdl_trigger();
  const int t = blockIdx.x;
  float* xr = x + (size_t)t * H;
  float ss = 0.f;
  for (int f = threadIdx.x; f < H; f += blockDim.x) {
    const float v = xr[f] + gather_partial(part, plan, H, t, f);
    xr[f] = v;
    ss += v * v;
  }
  ss = block_sum(ss, red);
  const float r = rsqrtf(ss / (float)H + eps);
  for (int f = threadIdx.x; f < H; f += blockDim.x) {
    const float y = xr[f] * r * to_f32(gain[f]);
    store_act(xn, (size_t)t * H + f, (size_t)kMaxT * H, y);
    if (hidden_out) hidden_out[(size_t)t * H + f] = y;
  }
}

cudaError_t launch_resid_norm(Model& m, const StreamK& plan, const void* gain, float* hidden_out, int T,
                              cudaStream_t st) {
  const auto& c = m.cfg;
  if (c.dtype == OOS_DTYPE_BF16)
    return launch(m.pdl, k_resid_norm<__nv_bfloat16>, dim3(T), dim3(256), 0, st, (const float*)m.ws.part, plan,
                  c.hidden, (const __nv_bfloat16*)gain, c.rms_eps, m.ws.x, (__nv_bfloat16*)m.ws.xn, hidden_out);
  return launch(m.pdl, k_resid_norm<float>, dim3(T), dim3(256), 0, st, (const float*)m.ws.part, plan, c.hidden,
                (const float*)gain, c.rms_eps, m.ws.x, (float*)m.ws.xn, hidden_out);
}

// ============================================================ SwiGLU
// act[t][i] = silu(gate) * up, gate/up = rows i and I + i of the stacked GEMM.
template <typename E>
__global__ void __launch_bounds__(256) k_silu_mul(const float* __restrict__ part, StreamK plan, int I,
                                                  E* __restrict__ act) {
  pdl_wait();
  pdl_trigger();
  const int t = blockIdx.y;
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < I) {
    const float g = gather_partial(part, plan, 2 * I, t, i);
    const float u = gather_partial(part, plan, 2 * I, t, I + i);
    store_act(act, (size_t)t * I + i, (size_t)kMaxT * I, g / (1.f + expf(-g)) * u);
  }
}

cudaError_t launch_silu_mul(Model& m, const StreamK& plan, int T, cudaStream_t st) {
  const auto& c = m.cfg;
  dim3 grid((c.intermediate + 255) / 256, T);
  if (c.dtype == OOS_DTYPE_BF16)
    return launch(m.pdl, k_silu_mul<__nv_bfloat16>, grid, dim3(256), 0, st, (const float*)m.ws.part, plan,
                  c.intermediate, (__nv_bfloat16*)m.ws.act);
  return launch(m.pdl, k_silu_mul<float>, grid, dim3(256), 0, st, (const float*)m.ws.part, plan, c.intermediate,
                (float*)m.ws.act);
}

// ============================================================ argmax merge + acceptance walk
// Running greedy state: largest logit, its (lowest) vocab id, second largest
// logit counted with multiplicity.
struct Top2 {
  float v1;
  int i1;
  float v2;
};
OOS_DEV Top2 top2_merge(Top2 a, Top2 b) {
  Top2 r;
  if (a.v1 > b.v1 || (a.v1 == b.v1 && a.i1 <= b.i1)) {
    r.v1 = a.v1;
    r.i1 = a.i1;
  } else {
    r.v1 = b.v1;
    r.i1 = b.i1;
  }
  r.v2 = fmaxf(fminf(a.v1, b.v1), fmaxf(a.v2, b.v2));
  return r;
}

// Greedy longest-prefix acceptance (Eq. 1; "Verify and commit") by one warp.
// ok(0) = 1; ok(i) = ok(parent) and token_i == argmax(parent).  The committed
// path ends at the deepest ok node (lowest id on ties); bonus = its argmax.
// Nodes at or past n_valid are padding of a fixed-size tree and never ok.
OOS_DEV void accept_walk_warp(const int32_t* tokens, const int32_t* parent, const int32_t* depth,
                              const int32_t* argmax, int T, int n_valid, bool bad, int32_t* len_out,
                              int32_t* nodes_out, int32_t* toks_out, int32_t* bonus_out) {
  const int lane = threadIdx.x & 31;
  if (bad) {
    for (int i = lane; i < T; i += 32) {
      nodes_out[i] = -1;
      toks_out[i] = -1;
    }
    if (lane == 0) {
      *len_out = 0;
      *bonus_out = -1;
    }
    return;
  }
  int best_key = 0x7fffffff;  // key = (kMaxT - depth) * 256 + node: min = deepest, then lowest id
  for (int i = lane; i < T; i += 32) {
    bool ok = i < n_valid;
    for (int a = i; ok && a != 0; a = parent[a]) {
      const int p = parent[a];
      if (tokens[a] != argmax[p]) {
        ok = false;
        break;
      }
    }
    if (ok) {
      const int key = (kMaxT - depth[i]) * 256 + i;
      best_key = key < best_key ? key : best_key;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const int other = __shfl_xor_sync(0xffffffffu, best_key, o);
    best_key = other < best_key ? other : best_key;
  }
  const int deepest = best_key & 255;
  const int len = depth[deepest] + 1;
  for (int j = len + lane; j < T; j += 32) {
    nodes_out[j] = -1;
    toks_out[j] = -1;
  }
  if (lane == 0) {
    for (int a = deepest; a >= 0; a = (a == 0 ? -1 : parent[a])) {
      nodes_out[depth[a]] = a;
      toks_out[depth[a]] = tokens[a];
    }
    *len_out = len;
    *bonus_out = argmax[deepest];
  }
}

__global__ void __launch_bounds__(1024) k_argmax_accept(const float* __restrict__ v1, const int32_t* __restrict__ i1,
                                                         const float* __restrict__ v2, int n_parts,
                                                         const int32_t* __restrict__ tokens,
                                                         const int32_t* __restrict__ parent,
                                                         const int32_t* __restrict__ depth, const uint32_t* status,
                                                         int T, const int32_t* __restrict__ n_valid_dev,
                                                         int32_t* argmax_ws, float* top1_ws, float* top2_ws,
                                                         int32_t* len, int32_t* nodes, int32_t* toks, int32_t* bonus,
                                                         int32_t* dbg_argmax, float* dbg_top1, float* dbg_top2) {
  __shared__ int32_t s_tok[kMaxT], s_par[kMaxT], s_dep[kMaxT], s_arg[kMaxT];
  pdl_wait();
  pdl_trigger();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  // one warp per node (32 warps); the merge is order independent (max with
  // lowest-id ties, multiset second max), so lanes take CTA states in any order
  for (int t = warp; t < T; t += nw) {
    Top2 r{-INFINITY, 0x7fffffff, -INFINITY};
#pragma unroll 4
    for (int c = lane; c < n_parts; c += 32) {
      const size_t k = (size_t)c * kMaxT + t;
      r = top2_merge(r, Top2{v1[k], i1[k], v2[k]});
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      Top2 y{__shfl_xor_sync(0xffffffffu, r.v1, o), __shfl_xor_sync(0xffffffffu, r.i1, o),
             __shfl_xor_sync(0xffffffffu, r.v2, o)};
      r = top2_merge(r, y);
    }
    if (lane == 0) {
      argmax_ws[t] = r.i1;
      top1_ws[t] = r.v1;
      top2_ws[t] = r.v2;
      if (dbg_argmax) dbg_argmax[t] = r.i1;
      if (dbg_top1) dbg_top1[t] = r.v1;
      if (dbg_top2) dbg_top2[t] = r.v2;
      s_arg[t] = r.i1;
    }
  }
  const int i = threadIdx.x;
  if (i < T) {
    s_tok[i] = tokens[i];
    s_par[i] = parent[i];
    s_dep[i] = depth[i];
  }
  __syncthreads();
  if (threadIdx.x < 32) {
    int n_valid = n_valid_dev ? *n_valid_dev : T;
    n_valid = n_valid < 1 ? 1 : (n_valid > T ? T : n_valid);
    // a malformed tree or a pipeline wait that gave up: no accepted path
    accept_walk_warp(s_tok, s_par, s_dep, s_arg, T, n_valid, (*status & (ST_TREE | ST_TIMEOUT)) != 0, len, nodes,
                     toks, bonus);
  }
}

cudaError_t launch_argmax_accept(Model& m, const int32_t* tokens, const int32_t* parent, int T, const int32_t* n_valid,
                                 int n_parts, int32_t* len, int32_t* nodes, int32_t* toks, int32_t* bonus,
                                 int32_t* dbg_argmax, float* dbg_top1, float* dbg_top2, cudaStream_t st) {
  return launch(m.pdl, k_argmax_accept, dim3(1), dim3(1024), 0, st, (const float*)m.ws.lm_v1,
                (const int32_t*)m.ws.lm_i, (const float*)m.ws.lm_v2, n_parts, tokens, parent,
                (const int32_t*)m.ws.depth, (const uint32_t*)m.ws.status, T, n_valid, m.ws.argmax, m.ws.top1,
                m.ws.top2, len, nodes, toks, bonus, dbg_argmax, dbg_top1, dbg_top2);
}

// standalone walk: validates the tree itself
__global__ void k_accept_walk(const int32_t* tokens, const int32_t* parent, const int32_t* argmax, int T,
                              int32_t* len, int32_t* nodes, int32_t* toks, int32_t* bonus, int32_t* status) {
  __shared__ int32_t s_tok[kMaxT], s_par[kMaxT], s_dep[kMaxT], s_arg[kMaxT];
  __shared__ int s_bad;
  const int i = threadIdx.x;
  if (i == 0) s_bad = 0;
  __syncthreads();
  if (i < T) {
    s_tok[i] = tokens[i];
    s_par[i] = parent[i];
    s_arg[i] = argmax[i];
    const bool ok = i == 0 ? s_par[i] == -1 : (s_par[i] >= 0 && s_par[i] < i);
    if (!ok) atomicOr(&s_bad, 1);
  }
  __syncthreads();
  if (i < T) {
    int d = 0;
    if (!s_bad)
      for (int a = i; a != 0; a = s_par[a]) ++d;
    s_dep[i] = d;
  }
  __syncthreads();
  if (i < 32) accept_walk_warp(s_tok, s_par, s_dep, s_arg, T, T, s_bad != 0, len, nodes, toks, bonus);
  if (i == 0) *status = s_bad ? OOS_ETREE : OOS_OK;
}

cudaError_t launch_accept_walk(const int32_t* tokens, const int32_t* parent, const int32_t* argmax, int T,
                               int32_t* len, int32_t* nodes, int32_t* toks, int32_t* bonus, int32_t* status,
                               cudaStream_t st) {
  k_accept_walk<<<1, kMaxT, 0, st>>>(tokens, parent, argmax, T, len, nodes, toks, bonus, status);
  return cudaGetLastError();
}

// ============================================================ KV compaction
// Slot ctx + j <- slot ctx + nodes[j] for j < len, per layer, for K and V.
// One block per (layer, K|V, kv head): all sources are staged in shared
// memory before any destination is written, so a source that is also a later
// destination is read before it is overwritten.
struct KvPtrs {
  void* k[kMaxLayers];
  void* v[kMaxLayers];
};

template <typename E>
__global__ void k_kv_compact(KvPtrs p, int nkv, int d, int ctx, const int32_t* __restrict__ ctx_dev,
                             const int32_t* __restrict__ nodes, const int32_t* __restrict__ len_ptr, int max_len) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  E* buf = reinterpret_cast<E*>(smem_raw);
  pdl_wait();
  pdl_trigger();
  if (ctx_dev) ctx = *ctx_dev;
  const int layer = blockIdx.x, which = blockIdx.y, g = blockIdx.z;
  E* base = (E*)(which == 0 ? p.k[layer] : p.v[layer]);
  int len = *len_ptr;
  len = len < 0 ? 0 : (len > max_len ? max_len : len);
  for (int e = threadIdx.x; e < len * d; e += blockDim.x) {
    const int j = e / d, c = e % d;
    const int src = nodes[j];
    if (src >= 0 && src < max_len) buf[e] = base[((size_t)(ctx + src) * nkv + g) * d + c];
  }
  __syncthreads();
  for (int e = threadIdx.x; e < len * d; e += blockDim.x) {
    const int j = e / d, c = e % d;
    const int src = nodes[j];
    if (src >= 0 && src < max_len) base[((size_t)(ctx + j) * nkv + g) * d + c] = buf[e];
  }
}

cudaError_t compact_setup() {
  cudaError_t e = cudaFuncSetAttribute(k_kv_compact<float>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       kMaxT * 128 * 4);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(k_kv_compact<__nv_bfloat16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              kMaxT * 128 * 2);
}

cudaError_t launch_kv_compact(Model& m, const oos_kv_cache& kv, int ctx, const int32_t* ctx_dev, const int32_t* nodes,
                              const int32_t* len, int max_len, cudaStream_t st) {
  const auto& c = m.cfg;
  KvPtrs p;
  for (int l = 0; l < c.n_layers; ++l) {
    p.k[l] = kv.k[l];
    p.v[l] = kv.v[l];
  }
  dim3 grid(c.n_layers, 2, c.n_kv_heads);
  const size_t smem = (size_t)max_len * c.head_dim * m.esize;
  if (c.dtype == OOS_DTYPE_BF16)
    return launch(m.pdl, k_kv_compact<__nv_bfloat16>, grid, dim3(256), smem, st, p, c.n_kv_heads, c.head_dim, ctx,
                  ctx_dev, nodes, len, max_len);
  return launch(m.pdl, k_kv_compact<float>, grid, dim3(256), smem, st, p, c.n_kv_heads, c.head_dim, ctx, ctx_dev,
                nodes, len, max_len);
}

}  // namespace oos
