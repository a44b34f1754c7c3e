// Multi-step decoding on the device: the ToolSpec loop (Section 2, "The
// ToolSpec decoding loop"; Section 4, "Verify and commit"; Section 5, #MAT)
// with the verifier of this library.
//
// One round: the next candidate tree from the request's hint bank, matched
// against everything committed so far (hint.cu: suffix match, hint lanes,
// prefix-tree packing), padded to a fixed node count; one verification of that
// tree, with the committed length and the real node count read from device
// memory; compaction of the accepted path's K/V; and the commit, which appends
// the accepted draft tokens and the bonus to the committed sequence (the
// bonus is the next round's root) and advances the committed length.  Every
// size the host needs is fixed, so a round is captured once as a CUDA graph
// and replayed, with no host round trip between rounds.
#include <string.h>

#include "common.cuh"
#include "internal.h"

namespace oos {

// state[0]: committed cache positions, state[1]: committed tokens, state[2]: rounds done
__global__ void k_decode_init(int32_t* state, int ctx, int n_committed) {
  state[0] = ctx;
  state[1] = n_committed;
  state[2] = 0;
}

// Append the round's accepted draft tokens (nodes 1 .. len-1 of the path) and
// the bonus; len tokens in all, the call's #MAT.  A round whose verification
// reported an error (len 0) commits nothing.
__global__ void k_decode_commit(int32_t* state, int32_t* committed, const int32_t* __restrict__ len_ptr,
                                const int32_t* __restrict__ toks, const int32_t* __restrict__ bonus,
                                int32_t* out_mat) {
  const int len = *len_ptr;
  const int n = state[1];
  for (int j = threadIdx.x; j < len; j += blockDim.x)
    committed[n + j] = j + 1 < len ? toks[j + 1] : *bonus;
  __syncthreads();
  if (threadIdx.x == 0) {
    out_mat[state[2]] = len;
    state[0] += len;
    state[1] = n + len;
    state[2] += 1;
  }
}

struct DecodeWs {
  void* hint_ws;
  int32_t *tok, *par, *T, *info, *len, *nodes, *toks, *bonus;
};

static size_t align256(size_t x) { return (x + 255) / 256 * 256; }

static size_t decode_ws_layout(long long bank_len, uint8_t* base, DecodeWs* d) {
  size_t off = 0;
  auto take = [&](size_t bytes) -> void* {
    void* p = base ? base + off : nullptr;
    off += align256(bytes);
    return p;
  };
  DecodeWs w;
  w.hint_ws = take(hint_workspace_bytes(bank_len));
  w.tok = (int32_t*)take(kMaxT * 4);
  w.par = (int32_t*)take(kMaxT * 4);
  w.T = (int32_t*)take(4);
  w.info = (int32_t*)take(3 * 4);
  w.len = (int32_t*)take(4);
  w.nodes = (int32_t*)take(kMaxT * 4);
  w.toks = (int32_t*)take(kMaxT * 4);
  w.bonus = (int32_t*)take(4);
  if (d) *d = w;
  return off;
}

#define OOS_TRY(x)                            \
  do {                                        \
    if ((x) != cudaSuccess) return OOS_ECUDA; \
  } while (0)

static int enqueue_round(Model& m, const oos_kv_cache* kv, int32_t* state, int32_t* committed, const int32_t* bank,
                         int bank_len, int eos, int max_lanes, int depth, int T_cap, int32_t* out_mat,
                         const DecodeWs& d, cudaStream_t st) {
  // the next tree: suffix match of the committed tokens (state[1] of them) in
  // the bank, hint lanes packed under the last committed token, padded to T_cap
  OOS_TRY(launch_hint_tree(bank, bank_len, eos, committed, 1, state + 1, nullptr, nullptr, 0, 1, max_lanes, depth,
                           T_cap, T_cap, d.hint_ws, d.tok, d.par, d.T, d.info, st));
  // verification at ctx = state[0]; only the d.T real nodes may be accepted
  const int rc = enqueue_verify_dev(m, kv, state, d.tok, d.par, T_cap, d.T, d.len, d.nodes, d.toks, d.bonus, st);
  if (rc != OOS_OK) return rc;
  OOS_TRY(launch_kv_compact(m, *kv, 0, state, d.nodes, d.len, T_cap, st));
  k_decode_commit<<<1, kMaxT, 0, st>>>(state, committed, d.len, d.toks, d.bonus, out_mat);
  OOS_TRY(cudaGetLastError());
  return OOS_OK;
}

}  // namespace oos

using namespace oos;

extern "C" {

size_t oos_decode_workspace_bytes(int32_t bank_len) {
  return bank_len < 1 ? 0 : decode_ws_layout(bank_len, nullptr, nullptr);
}

int oos_decode(oos_model* mp, const oos_kv_cache* kv, int32_t ctx_len, int32_t* committed, int32_t committed_len,
               int32_t committed_cap, const int32_t* bank, int32_t bank_len, int32_t eos, int32_t max_lanes,
               int32_t depth, int32_t max_nodes, int32_t n_rounds, int32_t* out_mat, int32_t* out_state,
               void* workspace, size_t ws_bytes, void* stream) {
  if (!mp || !kv || !committed || !bank || !out_mat || !out_state) return OOS_EINVAL;
  Model& m = *mp;
  if (kv->n_layers != m.cfg.n_layers || !kv->k || !kv->v || kv->capacity < 1) return OOS_EINVAL;
  for (int l = 0; l < kv->n_layers; ++l)
    if (!kv->k[l] || !kv->v[l]) return OOS_EINVAL;
  if (ctx_len < 0 || committed_len < 1 || bank_len < 1 || n_rounds < 1 || max_lanes < 0) return OOS_EINVAL;
  if (depth < 1 || depth > kMaxT || max_nodes < 1 || max_nodes > m.cfg.max_T) return OOS_EINVAL;
  // every round writes max_nodes tree slots and commits at most max_nodes tokens
  if ((long long)ctx_len + (long long)n_rounds * max_nodes > kv->capacity) return OOS_ECAPACITY;
  if ((long long)committed_len + (long long)n_rounds * max_nodes > committed_cap) return OOS_ECAPACITY;
  if (!workspace || ((uintptr_t)workspace & 255) || ws_bytes < decode_ws_layout(bank_len, nullptr, nullptr))
    return OOS_EWORKSPACE;
  DecodeWs d;
  decode_ws_layout(bank_len, (uint8_t*)workspace, &d);
  cudaStream_t st = (cudaStream_t)stream;
  k_decode_init<<<1, 1, 0, st>>>(out_state, ctx_len, committed_len);
  if (cudaGetLastError() != cudaSuccess) return OOS_ECUDA;
  if (!m.cfg.use_graph) {
    for (int r = 0; r < n_rounds; ++r) {
      const int rc = enqueue_round(m, kv, out_state, committed, bank, bank_len, eos, max_lanes, depth, max_nodes,
                                   out_mat, d, st);
      if (rc != OOS_OK) return rc;
    }
    return OOS_OK;
  }
  // one round as a graph, replayed n_rounds times: every argument of the
  // round is fixed, the changing values live in out_state
  cudaGraph_t graph = nullptr;
  cudaGraphExec_t exec = nullptr;
  if (cudaStreamBeginCapture(m.cap_stream, cudaStreamCaptureModeThreadLocal) != cudaSuccess) return OOS_ECUDA;
  int rc = enqueue_round(m, kv, out_state, committed, bank, bank_len, eos, max_lanes, depth, max_nodes, out_mat, d,
                         m.cap_stream);
  const cudaError_t ce = cudaStreamEndCapture(m.cap_stream, &graph);
  if (rc != OOS_OK || ce != cudaSuccess) {
    if (graph) cudaGraphDestroy(graph);
    return rc != OOS_OK ? rc : OOS_ECUDA;
  }
  if (cudaGraphInstantiate(&exec, graph, 0) != cudaSuccess) {
    cudaGraphDestroy(graph);
    return OOS_ECUDA;
  }
  cudaGraphDestroy(graph);
  for (int r = 0; r < n_rounds && rc == OOS_OK; ++r)
    if (cudaGraphLaunch(exec, st) != cudaSuccess) rc = OOS_ECUDA;
  // the launches are enqueued; the executable graph may be destroyed now
  cudaGraphExecDestroy(exec);
  return rc;
}

}  // extern "C"
