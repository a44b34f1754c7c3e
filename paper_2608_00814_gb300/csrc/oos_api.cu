// C ABI of the verify step (include/oos.h): argument validation, workspace
// carve-out, TMA descriptors, the per-call launch sequence and CUDA-graph
// replay.  Every step of the path runs in this library's kernels.
#include <math.h>
#include <stdlib.h>
#include <string.h>

#include <algorithm>
#include <new>
#include <vector>

#include "common.cuh"
#include "internal.h"

namespace oos {

static size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

StreamK make_streamk(int n_rows, int K, int n_sms, int tile_rows) {
  StreamK p;
  p.n_tiles = (n_rows + tile_rows - 1) / tile_rows;
  p.kbt = K / kBK;
  p.total = p.n_tiles * p.kbt;
  p.grid = std::min(std::min(n_sms, p.total), kMaxGridCTAs);
  return p;
}

StreamK make_single_slice(int n_rows) {
  StreamK p;
  p.n_tiles = (n_rows + kTile - 1) / kTile;
  p.kbt = 1;
  p.total = p.n_tiles;
  p.grid = p.n_tiles;
  return p;
}

static int lm_grid_for(const oos_model_config& c, int n_sms) {
  if (c.dtype == OOS_DTYPE_BF16)
    return std::min(std::min(n_sms, (c.vocab + kWorkRowsWide - 1) / kWorkRowsWide), kMaxGridCTAs);
  return std::max(1, std::min(std::min(2 * n_sms, (c.vocab + 15) / 16), kMaxGridCTAs));
}

size_t carve_workspace(const oos_model_config& c, int n_sms, uint8_t* base, Workspace* ws) {
  size_t off = 0;
  auto take = [&](size_t bytes) -> void* {
    off = align_up(off, 256);
    void* p = base ? base + off : nullptr;
    off += bytes;
    return p;
  };
  const size_t es = c.dtype == OOS_DTYPE_BF16 ? 2 : 4;
  const size_t H = c.hidden, I = c.intermediate, qd = (size_t)c.n_q_heads * c.head_dim;
  const size_t kvd = (size_t)c.n_kv_heads * c.head_dim;
  Workspace w;
  w.status = (uint32_t*)take(256);
  w.ctx = (int32_t*)take(256);
  w.depth = (int32_t*)take(kMaxT * 4);
  w.pos = (int32_t*)take(kMaxT * 4);
  w.anc = (unsigned long long*)take(kMaxT * 16);
  const size_t halves = c.dtype == OOS_DTYPE_BF16 ? 2 : 1;   // bf16: hi rows then lo rows
  w.x = (float*)take(kMaxT * H * 4);
  w.xn = take(halves * kMaxT * H * es);
  w.q = take(halves * kMaxT * qd * es);
  w.attn = take(halves * kMaxT * qd * es);
  w.act = take(halves * kMaxT * I * es);
  size_t pf = 0;
  const int Nq = (int)(qd + 2 * kvd);
  if (c.dtype == OOS_DTYPE_BF16) {
    const int rows[4] = {kTile, kTile, kWorkRowsWide, kTile};
    const StreamK ps[4] = {make_streamk(Nq, (int)H, n_sms, rows[0]), make_streamk((int)H, (int)qd, n_sms, rows[1]),
                           make_streamk((int)(2 * I), (int)H, n_sms, rows[2]),
                           make_streamk((int)H, (int)I, n_sms, rows[3])};
    for (int i = 0; i < 4; ++i) pf = std::max(pf, (size_t)ps[i].max_slices() * kMaxT * ps[i].n_tiles * rows[i]);
  } else {
    pf = (size_t)kMaxT * std::max(std::max((size_t)Nq, H), 2 * I);
  }
  w.part_floats = pf;
  w.part = (float*)take(pf * 4);
  const size_t lm = (size_t)kMaxGridCTAs * kMaxT;
  w.lm_v1 = (float*)take(lm * 4);
  w.lm_i = (int32_t*)take(lm * 4);
  w.lm_v2 = (float*)take(lm * 4);
  w.inv_freq = (double*)take((size_t)c.head_dim / 2 * 8);
  w.argmax = (int32_t*)take(kMaxT * 4);
  w.top1 = (float*)take(kMaxT * 4);
  w.top2 = (float*)take(kMaxT * 4);
  w.ss = (float*)take((size_t)kMaxSsChunks * kMaxT * 4);
  w.rope = (float2*)take((size_t)kMaxT * (c.head_dim / 2) * 8);
  w.cnt = (int*)take((size_t)c.n_layers * 4 * kCntPer * 4);
  w.chain_parent = (int32_t*)take(kMaxT * 4);
  w.pf_scratch = (int32_t*)take((2 + 2 * kMaxT) * 4);
  if (ws) *ws = w;
  return align_up(off, 256);
}

// Llama-3.1 rotary frequency rescaling of the pair rates theta^(-2m/d) (see
// oos_model_config): pairs of short wavelength keep their rate, long ones turn
// rope_factor times slower, the band between blends the two.
static void rope_rescale(std::vector<double>& inv, const oos_model_config& c) {
  const double F = c.rope_factor, lo = c.rope_low_freq_factor, hi = c.rope_high_freq_factor;
  const double L = (double)c.rope_orig_max_pos;
  for (double& f : inv) {
    const double wavelen = 2.0 * M_PI / f;
    if (wavelen < L / hi) continue;
    if (wavelen > L / lo) {
      f = f / F;
    } else {
      const double w = (L / wavelen - lo) / (hi - lo);
      f = (1.0 - w) * f / F + w * f;
    }
  }
}

static bool config_ok(const oos_model_config* c) {
  if (!c) return false;
  if (c->n_layers < 1 || c->n_layers > kMaxLayers) return false;
  if (c->hidden < 1 || c->n_q_heads < 1 || c->n_kv_heads < 1 || c->vocab < 1 || c->intermediate < 1) return false;
  if (c->n_q_heads % c->n_kv_heads) return false;
  if (c->head_dim < 2 || c->head_dim % 2 || c->head_dim > 128) return false;
  if (c->max_T < 1 || c->max_T > kMaxT) return false;
  if (c->dtype != OOS_DTYPE_F32 && c->dtype != OOS_DTYPE_BF16) return false;
  if (!(c->rms_eps >= 0.f) || !(c->rope_theta > 0.f)) return false;
  if (c->rope_factor > 1.f) {
    if (!(c->rope_low_freq_factor > 0.f) || !(c->rope_high_freq_factor > c->rope_low_freq_factor) ||
        c->rope_orig_max_pos < 1)
      return false;
  } else if (!(c->rope_factor == c->rope_factor)) {   // NaN
    return false;
  }
  return true;
}

static bool shape_supported(const oos_model_config* c) {
  if (c->kv_f16 && c->dtype != OOS_DTYPE_BF16) return false;   // FP16 caches: bf16 models only
  if (c->dtype == OOS_DTYPE_BF16) {
    if (c->head_dim != 128 || c->hidden % 128 || c->intermediate % 128) return false;
    if (c->hidden / 128 > kMaxSsChunks) return false;
    if (2 * c->intermediate / kWorkRowsWide > kCntPer || (c->n_q_heads + 2 * c->n_kv_heads) > kCntPer ||
        c->hidden / kTile > kCntPer)
      return false;
  }
  return true;
}

static int num_sms_current() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  return n;
}

static unsigned long long kv_hash(const oos_kv_cache* kv) {
  unsigned long long h = 1469598103934665603ull;
  for (int l = 0; l < kv->n_layers; ++l) {
    const unsigned long long a[2] = {(unsigned long long)(uintptr_t)kv->k[l], (unsigned long long)(uintptr_t)kv->v[l]};
    for (int i = 0; i < 2; ++i) {
      h ^= a[i];
      h *= 1099511628211ull;
    }
  }
  return h;
}

#define OOS_TRY(x)                         \
  do {                                     \
    if ((x) != cudaSuccess) return OOS_ECUDA; \
  } while (0)

// tree prep, embedding and every decoder layer of a tree on stream st: the
// K/V of the T nodes land in slots ctx.., the final-norm input in ws.x.  The
// committed length ctx comes from the host, or from device memory when ctx_dev
// is not null (then any value up to the cache capacity is allowed).
static int enqueue_layers(Model& m, const oos_kv_cache* kv, int ctx, const int32_t* ctx_dev, const int32_t* tokens,
                          const int32_t* parent, int T, float* hidden, cudaStream_t st) {
  const auto& c = m.cfg;
  const int L = c.n_layers;
  const int qd = c.n_q_heads * c.head_dim, kvd = c.n_kv_heads * c.head_dim;
  const int ctx_hint = ctx_dev ? kv->capacity - T : ctx;   // sizes the attention's key splits
  OOS_TRY(launch_tree_prep(m, tokens, parent, T, ctx, ctx_dev, st));
  if (c.dtype == OOS_DTYPE_BF16) OOS_TRY(launch_embed_tc(m, tokens, T, st));
  else OOS_TRY(launch_embed_norm(m, tokens, T, st));
  for (int l = 0; l < L; ++l) {
    const oos_layer_weights& W = m.layers[l];
    const void* next_gain = (l + 1 < L) ? m.layers[l + 1].attn_norm : m.w.final_norm;
    float* hid = (l + 1 < L) ? nullptr : hidden;
    if (c.dtype == OOS_DTYPE_BF16) {
      // five kernels per layer; every elementwise step runs in a GEMM epilogue
      OOS_TRY(launch_gemm_qkv(m, l, kv->k[l], kv->v[l], T, st));
      OOS_TRY(launch_attention(m, l, kv->k[l], kv->v[l], kv->capacity, ctx_hint, T, st));
      OOS_TRY(launch_gemm_o(m, l, T, st));
      OOS_TRY(launch_gemm_gu(m, l, T, st));
      OOS_TRY(launch_gemm_down(m, l, T, st));
    } else {
      OOS_TRY(launch_gemm_f32(m, W.w_q, W.w_k, W.w_v, qd, kvd, kvd, c.hidden, m.ws.xn, T, st));
      OOS_TRY(launch_qkv_post(m, l, m.p_qkv, kv->k[l], kv->v[l], T, st));
      OOS_TRY(launch_attention(m, l, kv->k[l], kv->v[l], kv->capacity, ctx_hint, T, st));
      OOS_TRY(launch_gemm_f32(m, W.w_o, nullptr, nullptr, c.hidden, 0, 0, qd, m.ws.attn, T, st));
      OOS_TRY(launch_resid_norm(m, m.p_o, W.mlp_norm, nullptr, T, st));
      OOS_TRY(launch_gemm_f32(m, W.w_gate, W.w_up, nullptr, c.intermediate, c.intermediate, 0, c.hidden, m.ws.xn, T,
                              st));
      OOS_TRY(launch_silu_mul(m, m.p_gu, T, st));
      OOS_TRY(launch_gemm_f32(m, W.w_down, nullptr, nullptr, c.hidden, 0, 0, c.intermediate, m.ws.act, T, st));
      OOS_TRY(launch_resid_norm(m, m.p_down, next_gain, hid, T, st));
    }
  }
  return OOS_OK;
}

// the whole verify step on stream st (ctx_dev, n_valid: see enqueue_verify_dev)
static int enqueue_verify(Model& m, const oos_kv_cache* kv, int ctx, const int32_t* ctx_dev, const int32_t* tokens,
                          const int32_t* parent, int T, const int32_t* n_valid, int32_t* len, int32_t* nodes,
                          int32_t* toks, int32_t* bonus, float* hidden, int32_t* dbg_arg, float* dbg_t1,
                          float* dbg_t2, cudaStream_t st) {
  const auto& c = m.cfg;
  const int rc = enqueue_layers(m, kv, ctx, ctx_dev, tokens, parent, T, hidden, st);
  if (rc != OOS_OK) return rc;
  if (c.dtype == OOS_DTYPE_BF16) {
    if (hidden) OOS_TRY(launch_final_hidden(m, hidden, T, st));
    OOS_TRY(launch_lm_head_tc(m, T, st));
  } else {
    OOS_TRY(launch_lm_head_f32(m, T, st));
  }
  OOS_TRY(launch_argmax_accept(m, tokens, parent, T, n_valid, m.lm_grid, len, nodes, toks, bonus, dbg_arg, dbg_t1,
                               dbg_t2, st));
  return OOS_OK;
}

int enqueue_verify_dev(Model& m, const oos_kv_cache* kv, const int32_t* ctx_dev, const int32_t* tokens,
                       const int32_t* parent, int T, const int32_t* n_valid, int32_t* len, int32_t* nodes,
                       int32_t* toks, int32_t* bonus, cudaStream_t st) {
  return enqueue_verify(m, kv, 0, ctx_dev, tokens, parent, T, n_valid, len, nodes, toks, bonus, nullptr, nullptr,
                        nullptr, nullptr, st);
}

// Prefill: the prompt as chains of at most max_T tokens.  In a chain node j's
// ancestors are nodes 0..j and its depth is j, so each chunk's tree pass is
// causal decoding of the chunk after everything before it, and node j's K/V
// land in their final slot ctx + off + j (no compaction).  Only the last chunk
// runs the LM head: the argmax of its last node is the greedy next token.
static int prefill_impl(Model& m, const oos_kv_cache* kv, int ctx, const int32_t* tokens, int n, int32_t* next_token,
                        cudaStream_t st) {
  const auto& c = m.cfg;
  int32_t* sc = m.ws.pf_scratch;
  for (int off = 0; off < n; off += c.max_T) {
    const int T = std::min(c.max_T, n - off);
    const int rc = enqueue_layers(m, kv, ctx + off, nullptr, tokens + off, m.ws.chain_parent, T, nullptr, st);
    if (rc != OOS_OK) return rc;
    if (off + T < n) continue;
    if (c.dtype == OOS_DTYPE_BF16) OOS_TRY(launch_lm_head_tc(m, T, st));
    else OOS_TRY(launch_lm_head_f32(m, T, st));
    OOS_TRY(launch_argmax_accept(m, tokens + off, m.ws.chain_parent, T, nullptr, m.lm_grid, sc, sc + 2,
                                 sc + 2 + kMaxT, sc + 1, nullptr, nullptr, nullptr, st));
    if (next_token) OOS_TRY(cudaMemcpyAsync(next_token, m.ws.argmax + (T - 1), 4, cudaMemcpyDeviceToDevice, st));
  }
  return OOS_OK;
}

static int verify_impl(oos_model* mp, const oos_kv_cache* kv, int32_t ctx, const int32_t* tokens,
                       const int32_t* parent, int32_t T, int32_t* len, int32_t* nodes, int32_t* toks, int32_t* bonus,
                       float* hidden, int32_t* dbg_arg, float* dbg_t1, float* dbg_t2, void* stream) {
  if (!mp || !kv || !tokens || !parent || !len || !nodes || !toks || !bonus) return OOS_EINVAL;
  Model& m = *mp;
  if (T < 1 || T > m.cfg.max_T || ctx < 0) return OOS_EINVAL;
  if (kv->n_layers != m.cfg.n_layers || !kv->k || !kv->v || kv->capacity < 1) return OOS_EINVAL;
  for (int l = 0; l < kv->n_layers; ++l)
    if (!kv->k[l] || !kv->v[l]) return OOS_EINVAL;
  if ((long long)ctx + T > kv->capacity) return OOS_ECAPACITY;
  cudaStream_t st = (cudaStream_t)stream;
  if (!m.cfg.use_graph)
    return enqueue_verify(m, kv, ctx, nullptr, tokens, parent, T, nullptr, len, nodes, toks, bonus, hidden, dbg_arg,
                          dbg_t1, dbg_t2, st);
  GraphKey key;
  key.kv_hash = kv_hash(kv);
  key.capacity = kv->capacity;
  key.splits = m.cfg.dtype == OOS_DTYPE_BF16 ? attn_splits(m, ctx, T) : 0;
  key.T = T;
  const void* io[10] = {tokens, parent, len, nodes, toks, bonus, hidden, dbg_arg, dbg_t1, dbg_t2};
  for (int i = 0; i < 10; ++i) key.io[i] = io[i];
  bool capture = !(m.have_graph && key == m.gkey);
  if (!capture && ctx != m.g_ctx) {
    // same graph at another committed length: only the tree-prep node changes
    if (set_tree_prep_ctx(m, m.gexec, m.prep_node, tokens, parent, T, ctx) == cudaSuccess) {
      m.g_ctx = ctx;
    } else {
      cudaGetLastError();
      capture = true;
    }
  }
  if (capture) {
    // a new shape or new buffers: capture again and instantiate afresh (the
    // tree-prep node handle must come from the graph the executable was made from)
    m.have_graph = false;
    if (m.gexec) cudaGraphExecDestroy(m.gexec);
    if (m.graph) cudaGraphDestroy(m.graph);
    m.gexec = nullptr;
    m.graph = nullptr;
    m.prep_node = nullptr;
    cudaGraph_t graph = nullptr;
    OOS_TRY(cudaStreamBeginCapture(m.cap_stream, cudaStreamCaptureModeThreadLocal));
    int rc = enqueue_verify(m, kv, ctx, nullptr, tokens, parent, T, nullptr, len, nodes, toks, bonus, hidden, dbg_arg,
                            dbg_t1, dbg_t2, m.cap_stream);
    cudaError_t ce = cudaStreamEndCapture(m.cap_stream, &graph);
    if (rc != OOS_OK || ce != cudaSuccess) {
      if (graph) cudaGraphDestroy(graph);
      return rc != OOS_OK ? rc : OOS_ECUDA;
    }
    cudaGraphNode_t prep = find_tree_prep_node(graph);
    if (!prep || cudaGraphInstantiate(&m.gexec, graph, 0) != cudaSuccess) {
      cudaGetLastError();
      cudaGraphDestroy(graph);
      m.gexec = nullptr;
      return OOS_ECUDA;
    }
    m.graph = graph;
    m.prep_node = prep;
    m.g_ctx = ctx;
    m.gkey = key;
    m.have_graph = true;
  }
  OOS_TRY(cudaGraphLaunch(m.gexec, st));
  return OOS_OK;
}

}  // namespace oos

using namespace oos;

extern "C" {

size_t oos_workspace_bytes(const oos_model_config* cfg) {
  if (!config_ok(cfg)) return 0;
  const int n = num_sms_current();
  if (n <= 0) return 0;
  return carve_workspace(*cfg, n, nullptr, nullptr);
}

int oos_model_create(const oos_model_config* cfg, const oos_weights* w, void* workspace, size_t ws_bytes,
                     oos_model** out) {
  if (!out) return OOS_EINVAL;
  *out = nullptr;
  if (!config_ok(cfg) || !w) return OOS_EINVAL;
  if (!shape_supported(cfg)) return OOS_EUNSUPPORTED;
  const oos_model_config& c = *cfg;
  if (!w->embed || !w->final_norm || !w->lm_head || !w->layers) return OOS_EINVAL;
  for (int l = 0; l < c.n_layers; ++l) {
    const oos_layer_weights& L = w->layers[l];
    if (!L.attn_norm || !L.w_q || !L.w_k || !L.w_v || !L.w_o || !L.mlp_norm || !L.w_gate || !L.w_up || !L.w_down)
      return OOS_EINVAL;
    if (c.qkv_bias && (!L.b_q || !L.b_k || !L.b_v)) return OOS_EINVAL;
    if (c.qk_norm && (!L.q_norm || !L.k_norm)) return OOS_EINVAL;
  }
  const int n_sms = num_sms_current();
  if (n_sms <= 0) return OOS_ECUDA;
  const size_t need = carve_workspace(c, n_sms, nullptr, nullptr);
  if (!workspace || ((uintptr_t)workspace & 255) || ws_bytes < need) return OOS_EWORKSPACE;

  oos_model* m = new (std::nothrow) oos_model();
  if (!m) return OOS_ECUDA;
  m->cfg = c;
  m->layers.assign(w->layers, w->layers + c.n_layers);
  m->w = *w;
  m->w.layers = m->layers.data();
  m->num_sms = n_sms;
  m->esize = c.dtype == OOS_DTYPE_BF16 ? 2 : 4;
  m->ws_bytes = need;
  carve_workspace(c, n_sms, (uint8_t*)workspace, &m->ws);
  const char* pdl_env = getenv("OOS_DISABLE_PDL");
  m->pdl = !(pdl_env && pdl_env[0] == '1');

  int rc = OOS_OK;
  do {
    if (cudaMemset(workspace, 0, need) != cudaSuccess) { rc = OOS_ECUDA; break; }
    const unsigned long long limit = kWaitLimitNs;
    if (cudaMemcpy(m->ws.status + kStatusWaitLimit, &limit, sizeof(limit), cudaMemcpyHostToDevice) != cudaSuccess) {
      rc = OOS_ECUDA;
      break;
    }
    std::vector<double> inv(c.head_dim / 2);
    for (int j = 0; j < c.head_dim / 2; ++j) inv[j] = pow((double)c.rope_theta, -2.0 * j / (double)c.head_dim);
    if (c.rope_factor > 1.f) rope_rescale(inv, c);
    if (cudaMemcpy(m->ws.inv_freq, inv.data(), inv.size() * 8, cudaMemcpyHostToDevice) != cudaSuccess) {
      rc = OOS_ECUDA;
      break;
    }
    std::vector<int32_t> chain(kMaxT);
    for (int i = 0; i < kMaxT; ++i) chain[i] = i - 1;
    if (cudaMemcpy(m->ws.chain_parent, chain.data(), kMaxT * 4, cudaMemcpyHostToDevice) != cudaSuccess) {
      rc = OOS_ECUDA;
      break;
    }
    if (gemm_setup() != cudaSuccess || attn_setup() != cudaSuccess || compact_setup() != cudaSuccess) {
      rc = OOS_ECUDA;
      break;
    }
    const int H = c.hidden, I = c.intermediate, qd = c.n_q_heads * c.head_dim, kvd = c.n_kv_heads * c.head_dim;
    m->lm_grid = lm_grid_for(c, n_sms);
    if (c.dtype == OOS_DTYPE_BF16) {
      auto mk = [&](GemmW& g, const void* const* ptrs, const int* rows, int nseg, int K, int interleave,
                    int tile_rows) -> bool {
        memset(&g, 0, sizeof(g));
        g.interleave2 = interleave;
        int tiles = 0, N = 0;
        for (int s = 0; s < nseg; ++s) {
          if (!encode_weight_map(&g.map[s], ptrs[s], rows[s], K)) return false;
          g.ptr[s] = ptrs[s];
          tiles += (rows[s] + kTile - 1) / kTile;
          g.seg_tiles[s] = tiles;
          N += rows[s];
        }
        for (int s = nseg; s < 3; ++s) g.seg_tiles[s] = tiles;
        g.n_seg = nseg;
        g.N = N;
        g.K = K;
        g.plan = make_streamk(N, K, n_sms, tile_rows);
        g.sub = tile_rows / kTile;
        g.round_robin = 0;
        return true;
      };
      bool ok = true;
      m->g_qkv.resize(c.n_layers);
      m->g_o.resize(c.n_layers);
      m->g_gu.resize(c.n_layers);
      m->g_down.resize(c.n_layers);
      for (int l = 0; l < c.n_layers && ok; ++l) {
        const oos_layer_weights& L = m->layers[l];
        const void* pq[3] = {L.w_q, L.w_k, L.w_v};
        const int rq[3] = {qd, kvd, kvd};
        const void* po[1] = {L.w_o};
        const int ro[1] = {H};
        const void* pg[2] = {L.w_gate, L.w_up};
        const int rg[2] = {I, I};
        const void* pd[1] = {L.w_down};
        const int rd[1] = {H};
        ok = mk(m->g_qkv[l], pq, rq, 3, H, 0, kTile) && mk(m->g_o[l], po, ro, 1, qd, 0, kTile) &&
             mk(m->g_gu[l], pg, rg, 2, H, 1, kWorkRowsWide) && mk(m->g_down[l], pd, rd, 1, I, 0, kTile);
      }
      const void* pl[1] = {c.vocab ? w->lm_head : nullptr};
      const int rl[1] = {c.vocab};
      ok = ok && mk(m->g_lm, pl, rl, 1, H, 0, kWorkRowsWide);
      m->g_lm.round_robin = 1;
      m->g_lm.plan.grid = m->lm_grid;
      const int boxes[4] = {16, 32, 64, 128};
      for (int b = 0; b < 4 && ok; ++b)
        ok = encode_act_map(&m->amap_xn[b], m->ws.xn, H, boxes[b]) &&
             encode_act_map(&m->amap_attn[b], m->ws.attn, qd, boxes[b]) &&
             encode_act_map(&m->amap_act[b], m->ws.act, I, boxes[b]);
      ok = ok && attn_encode_q_maps(*m);
      if (!ok) {
        rc = OOS_ECUDA;
        break;
      }
    } else {
      m->p_qkv = make_single_slice(qd + 2 * kvd);
      m->p_o = make_single_slice(H);
      m->p_gu = make_single_slice(2 * I);
      m->p_down = make_single_slice(H);
    }
    if (c.use_graph && cudaStreamCreateWithFlags(&m->cap_stream, cudaStreamNonBlocking) != cudaSuccess) {
      rc = OOS_ECUDA;
      break;
    }
  } while (0);
  if (rc != OOS_OK) {
    if (m->cap_stream) cudaStreamDestroy(m->cap_stream);
    delete m;
    return rc;
  }
  *out = m;
  return OOS_OK;
}

int oos_model_destroy(oos_model* m) {
  if (!m) return OOS_EINVAL;
  if (m->gexec) cudaGraphExecDestroy(m->gexec);
  if (m->graph) cudaGraphDestroy(m->graph);
  if (m->cap_stream) cudaStreamDestroy(m->cap_stream);
  delete m;
  return OOS_OK;
}

int oos_tree_verify(oos_model* m, const oos_kv_cache* kv, int32_t ctx_len, const int32_t* tree_tokens,
                    const int32_t* tree_parent, int32_t T, int32_t* out_accepted_len, int32_t* out_accepted_nodes,
                    int32_t* out_accepted_tokens, int32_t* out_bonus_token, void* stream) {
  return verify_impl(m, kv, ctx_len, tree_tokens, tree_parent, T, out_accepted_len, out_accepted_nodes,
                     out_accepted_tokens, out_bonus_token, nullptr, nullptr, nullptr, nullptr, stream);
}

int oos_prefill(oos_model* m, const oos_kv_cache* kv, int32_t ctx_len, const int32_t* tokens, int32_t n,
                int32_t* out_next_token, void* stream) {
  if (!m || !kv || !tokens || n < 1 || ctx_len < 0) return OOS_EINVAL;
  if (kv->n_layers != m->cfg.n_layers || !kv->k || !kv->v || kv->capacity < 1) return OOS_EINVAL;
  for (int l = 0; l < kv->n_layers; ++l)
    if (!kv->k[l] || !kv->v[l]) return OOS_EINVAL;
  if ((long long)ctx_len + n > kv->capacity) return OOS_ECAPACITY;
  return prefill_impl(*m, kv, ctx_len, tokens, n, out_next_token, (cudaStream_t)stream);
}

int oos_tree_verify_debug(oos_model* m, const oos_kv_cache* kv, int32_t ctx_len, const int32_t* tree_tokens,
                          const int32_t* tree_parent, int32_t T, int32_t* out_accepted_len,
                          int32_t* out_accepted_nodes, int32_t* out_accepted_tokens, int32_t* out_bonus_token,
                          float* out_final_hidden, int32_t* out_argmax, float* out_top1, float* out_top2,
                          void* stream) {
  return verify_impl(m, kv, ctx_len, tree_tokens, tree_parent, T, out_accepted_len, out_accepted_nodes,
                     out_accepted_tokens, out_bonus_token, out_final_hidden, out_argmax, out_top1, out_top2, stream);
}

int oos_kv_compact(oos_model* m, const oos_kv_cache* kv, int32_t ctx_len, const int32_t* accepted_nodes,
                   const int32_t* accepted_len, int32_t max_len, void* stream) {
  if (!m || !kv || !accepted_nodes || !accepted_len) return OOS_EINVAL;
  if (kv->n_layers != m->cfg.n_layers || !kv->k || !kv->v) return OOS_EINVAL;
  for (int l = 0; l < kv->n_layers; ++l)
    if (!kv->k[l] || !kv->v[l]) return OOS_EINVAL;
  if (ctx_len < 0 || max_len < 1 || max_len > kMaxT) return OOS_EINVAL;
  if ((long long)ctx_len + max_len > kv->capacity) return OOS_ECAPACITY;
  if (launch_kv_compact(*m, *kv, ctx_len, nullptr, accepted_nodes, accepted_len, max_len, (cudaStream_t)stream) !=
      cudaSuccess)
    return OOS_ECUDA;
  return OOS_OK;
}

int oos_accept_walk(const int32_t* tree_tokens, const int32_t* tree_parent, const int32_t* argmax, int32_t T,
                    int32_t* out_accepted_len, int32_t* out_accepted_nodes, int32_t* out_accepted_tokens,
                    int32_t* out_bonus_token, int32_t* out_status, void* stream) {
  if (!tree_tokens || !tree_parent || !argmax || !out_accepted_len || !out_accepted_nodes || !out_accepted_tokens ||
      !out_bonus_token || !out_status)
    return OOS_EINVAL;
  if (T < 1 || T > kMaxT) return OOS_EINVAL;
  if (launch_accept_walk(tree_tokens, tree_parent, argmax, T, out_accepted_len, out_accepted_nodes,
                         out_accepted_tokens, out_bonus_token, out_status, (cudaStream_t)stream) != cudaSuccess)
    return OOS_ECUDA;
  return OOS_OK;
}

int oos_launch_stage(oos_model* m, int32_t layer, int32_t stage, int32_t T, void* stream) {
  if (!m || T < 1 || T > m->cfg.max_T || stage < OOS_STAGE_QKV || stage > OOS_STAGE_LM_HEAD) return OOS_EINVAL;
  if (stage != OOS_STAGE_LM_HEAD && (layer < 0 || layer >= m->cfg.n_layers)) return OOS_EINVAL;
  cudaStream_t st = (cudaStream_t)stream;
  const auto& c = m->cfg;
  const int qd = c.n_q_heads * c.head_dim, kvd = c.n_kv_heads * c.head_dim;
  cudaError_t e;
  if (c.dtype == OOS_DTYPE_BF16) {
    switch (stage) {
      case OOS_STAGE_QKV: return OOS_EINVAL;   // its epilogue writes the KV cache
      case OOS_STAGE_O:
      case OOS_STAGE_GATE_UP:
      case OOS_STAGE_DOWN: {
        // a lone GEMM: its arrival counters start from zero as in a verify step
        const int kind = stage == OOS_STAGE_O ? 1 : stage == OOS_STAGE_GATE_UP ? 2 : 3;
        e = cudaMemsetAsync(gemm_counters(*m, layer, kind), 0, kCntPer * sizeof(int), st);
        if (e != cudaSuccess) break;
        e = stage == OOS_STAGE_O ? launch_gemm_o(*m, layer, T, st)
            : stage == OOS_STAGE_GATE_UP ? launch_gemm_gu(*m, layer, T, st)
                                         : launch_gemm_down(*m, layer, T, st);
        break;
      }
      default: e = launch_lm_head_tc(*m, T, st); break;
    }
  } else {
    const oos_layer_weights& W = m->layers[stage == OOS_STAGE_LM_HEAD ? 0 : layer];
    switch (stage) {
      case OOS_STAGE_QKV: e = launch_gemm_f32(*m, W.w_q, W.w_k, W.w_v, qd, kvd, kvd, c.hidden, m->ws.xn, T, st); break;
      case OOS_STAGE_O: e = launch_gemm_f32(*m, W.w_o, nullptr, nullptr, c.hidden, 0, 0, qd, m->ws.attn, T, st); break;
      case OOS_STAGE_GATE_UP:
        e = launch_gemm_f32(*m, W.w_gate, W.w_up, nullptr, c.intermediate, c.intermediate, 0, c.hidden, m->ws.xn, T,
                            st);
        break;
      case OOS_STAGE_DOWN:
        e = launch_gemm_f32(*m, W.w_down, nullptr, nullptr, c.hidden, 0, 0, c.intermediate, m->ws.act, T, st);
        break;
      default: e = launch_lm_head_f32(*m, T, st); break;
    }
  }
  return e == cudaSuccess ? OOS_OK : OOS_ECUDA;
}

int oos_launch_attention(oos_model* m, const oos_kv_cache* kv, int32_t layer, int32_t ctx_len, int32_t T,
                         void* stream) {
  if (!m || !kv || kv->n_layers != m->cfg.n_layers || !kv->k || !kv->v) return OOS_EINVAL;
  if (layer < 0 || layer >= m->cfg.n_layers || !kv->k[layer] || !kv->v[layer]) return OOS_EINVAL;
  if (T < 1 || T > m->cfg.max_T || ctx_len < 0) return OOS_EINVAL;
  if ((long long)ctx_len + T > kv->capacity) return OOS_ECAPACITY;
  // the kernel reads the step's committed length from the workspace
  cudaStream_t st = (cudaStream_t)stream;
  const int32_t c32 = ctx_len;
  if (cudaMemcpyAsync(m->ws.ctx, &c32, sizeof(c32), cudaMemcpyHostToDevice, st) != cudaSuccess) return OOS_ECUDA;
  return launch_attention(*m, layer, kv->k[layer], kv->v[layer], kv->capacity, ctx_len, T, st) == cudaSuccess
             ? OOS_OK
             : OOS_ECUDA;
}

int oos_set_wait_limit(oos_model* m, uint64_t limit_ns, void* stream) {
  if (!m) return OOS_EINVAL;
  if (limit_ns == 0 || limit_ns > kWaitLimitNs) limit_ns = kWaitLimitNs;
  const unsigned long long v = limit_ns;
  cudaStream_t st = (cudaStream_t)stream;
  if (cudaMemcpyAsync(m->ws.status + kStatusWaitLimit, &v, sizeof(v), cudaMemcpyHostToDevice, st) != cudaSuccess)
    return OOS_ECUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return OOS_ECUDA;
  return OOS_OK;
}

int oos_last_status(oos_model* m, void* stream) {
  if (!m) return OOS_EINVAL;
  uint32_t s = 0;
  cudaStream_t st = (cudaStream_t)stream;
  if (cudaMemcpyAsync(&s, m->ws.status, 4, cudaMemcpyDeviceToHost, st) != cudaSuccess) return OOS_ECUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return OOS_ECUDA;
  if (s & ST_TIMEOUT) return OOS_ETIMEOUT;
  if (s & ST_TREE) return OOS_ETREE;
  return OOS_OK;
}

const char* oos_status_string(int code) {
  switch (code) {
    case OOS_OK: return "ok";
    case OOS_EINVAL: return "invalid argument";
    case OOS_ECAPACITY: return "ctx_len + T exceeds the KV cache capacity";
    case OOS_ECUDA: return "CUDA call failed";
    case OOS_ETREE: return "malformed tree (parent not parents-first, or token outside the vocabulary)";
    case OOS_ETIMEOUT: return "device pipeline wait exceeded its limit";
    case OOS_EUNSUPPORTED: return "model shape not supported by the kernels";
    case OOS_EWORKSPACE: return "workspace missing, misaligned or too small";
    default: return "unknown status";
  }
}

}  // extern "C"
