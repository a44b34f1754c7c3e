// Host-side model handle, workspace carve-out and kernel launchers.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>
#include <vector>

#include "oos.h"

namespace oos {

constexpr int kMaxT = 128;          // largest tree (ancestor sets are 128-bit masks)
constexpr int kTile = 128;          // weight rows per MMA (tcgen05 M)
constexpr int kWorkRowsWide = 256;  // weight rows per work tile of the gate/up GEMM and LM head
constexpr int kBK = 64;             // reduction elements per pipeline stage (128 bytes of bf16)
constexpr int kMaxLayers = 128;
constexpr int kMaxGridCTAs = 1024;  // upper bound on CTAs of a stream-K GEMM / LM head
constexpr int kMaxSsChunks = 64;    // hidden <= 8192: RMSNorm partial sums per 128 features
constexpr int kCntPer = 256;        // arrival counters per (layer, GEMM kind): one per work tile

// Stream-K partition of a weight GEMM: the (tile, k-block) units of all tiles,
// tile-major, are cut into `grid` contiguous equal ranges, one per CTA.  CTA c
// owns units [c*total/grid, (c+1)*total/grid).  Each CTA writes one fp32
// partial tile per tile it touches, into slice (c - first contributor of the
// tile); a reduce kernel adds the slices in slice order (deterministic).
struct StreamK {
  int n_tiles;
  int kbt;     // k-blocks per tile
  int total;   // n_tiles * kbt
  int grid;    // CTAs
  __host__ __device__ int cta_of_unit(long long u) const {
    // largest c with floor(c*total/grid) <= u
    return (int)(((u + 1) * (long long)grid + total - 1) / total) - 1;
  }
  __host__ __device__ void contributors(int tile, int& c0, int& c1) const {
    c0 = cta_of_unit((long long)tile * kbt);
    c1 = cta_of_unit((long long)tile * kbt + kbt - 1);
  }
  int max_slices() const {
    int m = 1;
    for (int t = 0; t < n_tiles; ++t) {
      int a, b;
      contributors(t, a, b);
      m = (b - a + 1) > m ? (b - a + 1) : m;
    }
    return m;
  }
};

StreamK make_streamk(int n_rows, int K, int n_sms, int tile_rows);
StreamK make_single_slice(int n_rows);   // one contributor per tile (CUDA-core GEMM)

// One weight GEMM of the bf16 path: up to three row-stacked segments (q|k|v,
// gate|up), each with its own TMA descriptor.
struct GemmW {
  CUtensorMap map[3];
  const void* ptr[3];
  int seg_tiles[3];   // cumulative tile counts at the end of each segment
  int n_seg;
  int interleave2;    // gate/up: tiles alternate between the two segments
  int sub;            // 128-row MMA subtiles per stream-K work tile (1 or 2)
  int round_robin;    // LM head: whole work tiles dealt round-robin instead of stream-K
  int N, K;
  StreamK plan;
};

struct Workspace {
  uint32_t* status;
  int32_t* ctx;              // committed length of the current step (written by tree preparation)
  int32_t* depth;
  int32_t* pos;
  unsigned long long* anc;   // [kMaxT][2]
  float* x;                  // residual stream, fp32 [kMaxT][H]
  void* xn;                  // normalised GEMM input [kMaxT][H] (model dtype)
  void* q;                   // [kMaxT][nq][d]
  void* attn;                // attention output [kMaxT][nq*d]
  void* act;                 // SwiGLU activation [kMaxT][I]
  float* part;               // GEMM partial slices
  size_t part_floats;
  float* lm_v1;              // LM-head partial states [kMaxGridCTAs][kMaxT]
  int32_t* lm_i;
  float* lm_v2;
  double* inv_freq;          // RoPE frequencies theta^(-2j/d), j < d/2
  int32_t* argmax;           // [kMaxT]
  float* top1;
  float* top2;
  float* ss;                 // sum of x^2 per 128-feature chunk [kMaxSsChunks][kMaxT] (bf16 path)
  float2* rope;              // (cos, sin) per node and rotary pair [kMaxT][d/2] (bf16 path)
  int* cnt;                  // GEMM arrival counters [layer][4 kinds][kCntPer], zeroed at every step start
  int32_t* chain_parent;     // [kMaxT]: -1, 0, 1, ... (the chains a prefill runs as trees)
  int32_t* pf_scratch;       // prefill's unused accept outputs: len, bonus, nodes[kMaxT], tokens[kMaxT]
};

// shape + addresses a captured verify graph was recorded with.  The committed
// length is not part of it: only the tree-prep kernel takes it as an argument
// (every later kernel reads it from ws.ctx), so a call at another length
// updates that one node.  What the length does decide on the host, the
// attention's key-split count, is.
struct GraphKey {
  unsigned long long kv_hash;   // FNV-1a over every layer's K and V pointer
  int capacity, splits, T;
  const void* io[10];
  bool operator==(const GraphKey& o) const {
    if (kv_hash != o.kv_hash || capacity != o.capacity || splits != o.splits || T != o.T) return false;
    for (int i = 0; i < 10; ++i)
      if (io[i] != o.io[i]) return false;
    return true;
  }
};

struct Model {
  oos_model_config cfg;
  std::vector<oos_layer_weights> layers;
  oos_weights w;
  int num_sms;
  int esize;            // bytes per weight / activation element
  Workspace ws;
  size_t ws_bytes;
  bool pdl = true;
  // bf16 tensor-core path
  std::vector<GemmW> g_qkv, g_o, g_gu, g_down;
  GemmW g_lm;
  CUtensorMap amap_xn[4], amap_attn[4], amap_act[4];  // per N-tile variant 16/32/64/128
  CUtensorMap qmap_hi, qmap_lo;   // attention: q rows of one kv head, (d, head in group, kv head, node)
  // attention: the K/V cache maps encoded per layer over the whole capacity
  // (re-encoded only when the cache buffers change)
  struct KvMaps {
    const void* k = nullptr;
    const void* v = nullptr;
    int extent = -1;
    CUtensorMap kmap, vmap;
  };
  std::vector<KvMaps> kv_maps;
  int lm_grid;
  // fp32 path plans (one slice)
  StreamK p_qkv, p_o, p_gu, p_down;
  // CUDA graph of the last call shape
  cudaStream_t cap_stream = nullptr;
  cudaGraph_t graph = nullptr;          // the graph gexec was instantiated from
  cudaGraphExec_t gexec = nullptr;
  cudaGraphNode_t prep_node = nullptr;  // its tree-prep kernel node
  int g_ctx = -1;                       // committed length that node was last given
  GraphKey gkey{};
  bool have_graph = false;
};

size_t carve_workspace(const oos_model_config& c, int n_sms, uint8_t* base, Workspace* ws);

// launch with or without programmatic dependent launch (PDL)
template <typename... KArgs, typename... Args>
inline cudaError_t launch(bool pdl, void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                          cudaStream_t st, Args&&... args) {
  cudaLaunchConfig_t lc = {};
  lc.gridDim = grid;
  lc.blockDim = block;
  lc.dynamicSmemBytes = smem;
  lc.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  lc.attrs = attr;
  lc.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&lc, kernel, std::forward<Args>(args)...);
}

// ---- small kernels (small.cu)
// ctx from the host, or from device memory when ctx_dev is not null
cudaError_t launch_tree_prep(Model& m, const int32_t* tokens, const int32_t* parent, int T, int ctx,
                             const int32_t* ctx_dev, cudaStream_t st);
// the tree-prep kernel node of a captured graph, and a new committed length for it
cudaGraphNode_t find_tree_prep_node(cudaGraph_t g);
cudaError_t set_tree_prep_ctx(Model& m, cudaGraphExec_t ex, cudaGraphNode_t node, const int32_t* tokens,
                              const int32_t* parent, int T, int ctx);
cudaError_t launch_embed_norm(Model& m, const int32_t* tokens, int T, cudaStream_t st);
cudaError_t launch_embed_tc(Model& m, const int32_t* tokens, int T, cudaStream_t st);
cudaError_t launch_final_hidden(Model& m, float* hidden, int T, cudaStream_t st);
cudaError_t launch_qkv_post(Model& m, int layer, const StreamK& plan, void* kc, void* vc, int T, cudaStream_t st);
cudaError_t launch_resid_norm(Model& m, const StreamK& plan, const void* gain, float* hidden_out, int T,
                              cudaStream_t st);
cudaError_t launch_silu_mul(Model& m, const StreamK& plan, int T, cudaStream_t st);
// n_valid: DEVICE count of real nodes (the rest is padding, never accepted), or nullptr for T
cudaError_t launch_argmax_accept(Model& m, const int32_t* tokens, const int32_t* parent, int T, const int32_t* n_valid,
                                 int n_parts, int32_t* len, int32_t* nodes, int32_t* toks, int32_t* bonus,
                                 int32_t* dbg_argmax, float* dbg_top1, float* dbg_top2, cudaStream_t st);
cudaError_t launch_kv_compact(Model& m, const oos_kv_cache& kv, int ctx, const int32_t* ctx_dev, const int32_t* nodes,
                              const int32_t* len, int max_len, cudaStream_t st);
cudaError_t compact_setup();
cudaError_t launch_accept_walk(const int32_t* tokens, const int32_t* parent, const int32_t* argmax, int T,
                               int32_t* len, int32_t* nodes, int32_t* toks, int32_t* bonus, int32_t* status,
                               cudaStream_t st);

// ---- GEMMs (gemm.cu)
bool encode_weight_map(CUtensorMap* map, const void* ptr, int rows, int K);
// 16-bit (bf16, or binary16 when f16) tensor map with 128-byte swizzle: dims[0]
// contiguous, strides[i] = bytes between consecutive indices of dim i + 1, box[]
// elements per dim
bool encode_bf16_map(CUtensorMap* map, const void* ptr, int rank, const uint64_t* dims, const uint64_t* strides,
                     const uint32_t* box, bool f16 = false);
bool encode_act_map(CUtensorMap* map, const void* ptr, int K, int box_rows);
int bn_index(int T);   // N-tile variant for T tree nodes: 0..3 -> 16/32/64/128
cudaError_t gemm_setup();
cudaError_t launch_gemm_qkv(Model& m, int layer, void* kc, void* vc, int T, cudaStream_t st);
cudaError_t launch_gemm_o(Model& m, int layer, int T, cudaStream_t st);
cudaError_t launch_gemm_gu(Model& m, int layer, int T, cudaStream_t st);
cudaError_t launch_gemm_down(Model& m, int layer, int T, cudaStream_t st);
cudaError_t launch_lm_head_tc(Model& m, int T, cudaStream_t st);
int* gemm_counters(Model& m, int layer, int kind);   // kind 0 qkv, 1 o, 2 gate/up, 3 down
cudaError_t launch_gemm_f32(Model& m, const void* w0, const void* w1, const void* w2, int rows0, int rows1,
                            int rows2, int K, const void* x, int T, cudaStream_t st);
cudaError_t launch_lm_head_f32(Model& m, int T, cudaStream_t st);

// ---- verify step with the committed length and the count of real nodes in
// device memory (oos_api.cu): tokens/parent hold T nodes of which *n_valid are
// real (the rest is padding that is never accepted); ctx_dev may be anything
// up to the cache capacity minus T
int enqueue_verify_dev(Model& m, const oos_kv_cache* kv, const int32_t* ctx_dev, const int32_t* tokens,
                       const int32_t* parent, int T, const int32_t* n_valid, int32_t* len, int32_t* nodes,
                       int32_t* toks, int32_t* bonus, cudaStream_t st);

// ---- hint-bank candidate step (hint.cu)
size_t hint_workspace_bytes(long long bank_len);
// prefix_len_dev: DEVICE prefix length (or nullptr for prefix_len); pad_to: write
// padding nodes up to this count (0: none)
cudaError_t launch_hint_tree(const int32_t* bank, int N, int eos, const int32_t* prefix, int prefix_len,
                             const int32_t* prefix_len_dev, const int32_t* native, const int32_t* native_len,
                             int n_native, int native_stride, int max_lanes, int depth, int max_nodes, int pad_to,
                             void* ws, int32_t* out_tok, int32_t* out_par, int32_t* out_T, int32_t* out_info,
                             cudaStream_t st);

// ---- attention (attn.cu)
cudaError_t attn_setup();
int attn_nodes_per_block(int group);   // tree nodes per attention block (x group q heads <= 128 rows)
bool attn_encode_q_maps(Model& m);     // TMA maps of the q buffer (bf16 path), at model creation
// the step's ctx comes from the workspace; ctx here only sizes the key splits
cudaError_t launch_attention(Model& m, int layer, const void* kc, const void* vc, int capacity, int ctx, int T,
                             cudaStream_t st);
int attn_splits(Model& m, int ctx_hint, int T);

}  // namespace oos

// the C handle of include/oos.h is the host-side model
struct oos_model : public oos::Model {};
