/*
 * oos.h -- C ABI of the GB300 tree-verification step.
 *
 * The step is the target verifier of OoO-Spec (arXiv 2608.00814):
 *   - Eq. 1 ("Target authority"): under greedy decoding the committed token is
 *     y_t = argmax_v p_T(v | x, y_<t); only the target extends the output.
 *   - Sec. "Target-Only Verification and Recovery", "Verify and commit": the
 *     candidate tree is evaluated in ONE forward pass of the target, the
 *     longest prefix allowed by the greedy rule is committed, the first
 *     mismatch is replaced by the target's own next token, and only states on
 *     the accepted path enter the committed KV cache.
 *   - Sec. "Background" (the ToolSpec loop): each round packs candidates into
 *     a tree, the target commits the longest approved prefix and the next
 *     tree is built from all committed tokens.
 *
 * Readings of what the paper leaves open (the verifier implements exactly
 * these):
 *   - Node 0 of a tree is the ROOT: the last committed token, whose K/V is not
 *     cached yet.  It is always accepted.  Nodes are numbered parents-first:
 *     parent[0] == -1 and 0 <= parent[i] < i.
 *   - Node i attends to the ctx_len committed cache positions and to its own
 *     ancestors (itself included); its RoPE position is ctx_len + depth(i).
 *   - A draft node is accepted when its parent is accepted and its token equals
 *     the target's argmax at the parent.  The committed path is root -> the
 *     deepest accepted node (lowest node id among equally deep ones).  The
 *     bonus token is the target's argmax at that node.  Argmax ties go to the
 *     lowest vocabulary id.
 *   - The decoder is a pre-norm Llama/Qwen block: RMSNorm, q/k/v projections
 *     (optional bias), optional per-head q/k RMSNorm before RoPE (Qwen3),
 *     rotate-half RoPE, grouped-query attention, output projection, RMSNorm,
 *     SwiGLU MLP (down(silu(gate h) * up h)), final RMSNorm, LM head.
 *
 * Conventions for every entry point:
 *   - Pointers marked DEVICE are CUDA device addresses on the current device;
 *     HOST pointers are ordinary host memory read during the call only.
 *   - The caller owns every buffer: weights, KV cache, inputs, outputs and the
 *     workspace.  The library allocates no device memory; oos_model_create
 *     allocates the small host-side handle (and a CUDA stream and events used
 *     for graph capture).
 *   - Work is enqueued on `stream` (a cudaStream_t passed as void*; NULL is the
 *     legacy default stream) and runs asynchronously; nothing here blocks the
 *     host except oos_last_status.
 *   - Matrices are row-major in the PyTorch nn.Linear layout [out, in];
 *     element type per oos_model_config.dtype (fp32 or bf16).  Norm gains and
 *     biases use the same element type.
 *   - Return value: OOS_OK (0) or a negative OOS_E* code.  Host-side argument
 *     errors are returned before anything is enqueued.  Errors that only the
 *     device can see (a malformed tree, an out-of-range token, a pipeline wait
 *     that ran out of time) are recorded in a device status word of the model
 *     and reported by oos_last_status; on such an error the verify outputs
 *     hold accepted_len = 0.
 */
#ifndef OOS_H
#define OOS_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes ---------------------------------------------------- */
#define OOS_OK 0
#define OOS_EINVAL (-1)        /* bad argument: NULL, T outside [1, max_T], ctx_len < 0, shape mismatch */
#define OOS_ECAPACITY (-2)     /* ctx_len + T exceeds the KV cache capacity */
#define OOS_ECUDA (-3)         /* a CUDA runtime or driver call failed */
#define OOS_ETREE (-4)         /* parent[] is not a parents-first tree, or a token is outside [0, vocab) */
#define OOS_ETIMEOUT (-5)      /* a device wait exceeded its limit; outputs are not valid and the handle
                                  must be destroyed and created again */
#define OOS_EUNSUPPORTED (-6)  /* shape outside what the kernels handle (see oos_model_create) */
#define OOS_EWORKSPACE (-7)    /* workspace NULL, misaligned (256 B) or smaller than oos_workspace_bytes */

#define OOS_DTYPE_F32 0
#define OOS_DTYPE_BF16 1

/* Model shape.  Supported: dtype BF16 with head_dim 128, hidden, q_dim and
 * intermediate multiples of 128 (tcgen05 path); dtype F32 with head_dim <= 128
 * even (CUDA-core path, meant for small models).  n_q_heads % n_kv_heads == 0,
 * n_layers <= 128, 1 <= max_T <= 128. */
typedef struct {
    int32_t n_layers;
    int32_t hidden;        /* H */
    int32_t n_q_heads;     /* nq */
    int32_t n_kv_heads;    /* nkv */
    int32_t head_dim;      /* d */
    int32_t intermediate;  /* I (SwiGLU width) */
    int32_t vocab;         /* V */
    int32_t dtype;         /* OOS_DTYPE_F32 or OOS_DTYPE_BF16: weights, KV cache, gains, biases */
    int32_t qk_norm;       /* nonzero: per-head RMSNorm of q and k before RoPE (Qwen3) */
    int32_t qkv_bias;      /* nonzero: bias on the q, k, v projections (Qwen2.5) */
    float rms_eps;
    float rope_theta;      /* RoPE base; pair (m, m + d/2) turns by pos * theta^(-2m/d) */
    int32_t max_T;         /* largest tree this handle verifies, 1..128 */
    int32_t use_graph;     /* nonzero: oos_tree_verify replays one captured CUDA graph while the
                              cache buffers, T, the I/O pointers and the attention's key-split
                              count repeat; a new committed length updates only the graph's
                              tree-preparation node (the other kernels read it from the
                              workspace); anything else is captured again */
    /* Rotary frequency rescaling of Llama-3.1 targets (the paper's Llama-3.1-8B),
     * as published with that model.  With factor F > 1, low-frequency factor lo,
     * high-frequency factor hi (hi > lo > 0) and original context L > 0, the
     * rate f = theta^(-2m/d) of pair m, of wavelength 2 pi / f, becomes
     *   f            when the wavelength is below L / hi,
     *   f / F        when it is above L / lo,
     *   (1 - w) f / F + w f,  w = (L / wavelength - lo) / (hi - lo), otherwise.
     * rope_factor <= 1 (0 when zero-initialised): no rescaling, the other three
     * fields are ignored.  Invalid values make oos_model_create fail with
     * OOS_EINVAL. */
    float rope_factor;
    float rope_low_freq_factor;
    float rope_high_freq_factor;
    int32_t rope_orig_max_pos;
    /* Nonzero: the KV cache holds IEEE binary16 (round to nearest even)
     * instead of the model dtype -- the FP16 cache backend of the paper's
     * Qwen2.5 and Llama runs ("Targets, Workloads, and Protocol").  bf16
     * models only (OOS_EUNSUPPORTED otherwise).  Every K/V a node attends to,
     * cached or written by the tree pass, is then binary16, and the attention
     * products run in f16. */
    int32_t kv_f16;
} oos_model_config;

/* Per-layer weights, all DEVICE pointers. */
typedef struct {
    const void* attn_norm;  /* [H] */
    const void* w_q;        /* [nq*d, H] */
    const void* w_k;        /* [nkv*d, H] */
    const void* w_v;        /* [nkv*d, H] */
    const void* b_q;        /* [nq*d]  or NULL (required iff qkv_bias) */
    const void* b_k;        /* [nkv*d] or NULL */
    const void* b_v;        /* [nkv*d] or NULL */
    const void* q_norm;     /* [d] or NULL (required iff qk_norm) */
    const void* k_norm;     /* [d] or NULL */
    const void* w_o;        /* [H, nq*d] */
    const void* mlp_norm;   /* [H] */
    const void* w_gate;     /* [I, H] */
    const void* w_up;       /* [I, H] */
    const void* w_down;     /* [H, I] */
} oos_layer_weights;

typedef struct {
    const void* embed;               /* DEVICE [V, H] */
    const void* final_norm;          /* DEVICE [H] */
    const void* lm_head;             /* DEVICE [V, H]; may equal embed (tied embeddings) */
    const oos_layer_weights* layers; /* HOST array of n_layers entries, copied by oos_model_create */
} oos_weights;

/* Committed KV cache: per layer one K and one V buffer of `capacity` slots.
 * Slot p holds the post-RoPE K (resp. V) of committed position p for all
 * kv heads: layout [capacity][nkv][d], element type = model dtype, or
 * binary16 with oos_model_config.kv_f16.  During
 * oos_tree_verify the tree's K/V are written to slots ctx_len .. ctx_len+T-1;
 * oos_kv_compact then moves the accepted path to ctx_len .. ctx_len+len-1. */
typedef struct {
    int32_t n_layers;
    int32_t capacity;
    void* const* k;   /* HOST array of n_layers DEVICE pointers */
    void* const* v;   /* HOST array of n_layers DEVICE pointers */
} oos_kv_cache;

typedef struct oos_model oos_model;

/* Bytes of DEVICE workspace one model handle needs (depends on the shape,
 * max_T and the current device's SM count).  Returns 0 on a bad config. */
size_t oos_workspace_bytes(const oos_model_config* cfg);

/* Validate the shape, copy the weight pointers, carve the caller's workspace
 * (DEVICE, >= oos_workspace_bytes, 256-byte aligned; owned by the caller and
 * bound to the handle until oos_model_destroy) and encode the TMA descriptors
 * of every weight matrix.  Weights must stay valid while the handle lives.
 * Uses the current CUDA device. */
int oos_model_create(const oos_model_config* cfg, const oos_weights* w, void* workspace,
                     size_t ws_bytes, oos_model** out);

int oos_model_destroy(oos_model* m);

/* Hint-bank candidate step: the next verification tree (Section 4, "Suffix
 * matching" and "Candidate boundary"; the tree is Merge_B of the hint lanes and
 * the verifier's native lanes).
 *   bank          DEVICE int32[bank_len]: the tokenised views joined by eos.
 *   prefix        DEVICE int32[prefix_len] (>= 1): the committed prefix y; its
 *                 last token is the tree's root, its last 7 tokens are matched.
 *   For n = min(7, prefix_len) down to 1, the length-n suffix of y is searched
 *   in the bank; an occurrence counts only when a non-eos token follows it, and
 *   the longest n with a counted occurrence is used.  Each of its occurrences,
 *   in bank order, proposes a lane: up to `depth` tokens after it, cut before
 *   an eos.  The native lanes follow: DEVICE int32[n_native][native_stride]
 *   with lengths native_len[n_native] (cut to depth), NULL when n_native == 0.
 *   Lanes are merged into a prefix tree rooted at y's last token, a node
 *   numbered when created (parents first); a lane counts towards max_lanes only
 *   when it creates a node; at most max_nodes nodes (1..128), depth 1..128.
 *   workspace     DEVICE, >= oos_hint_workspace_bytes(bank_len) (0 for bank_len < 1),
 *                 256-byte aligned; owned by the caller, scratch for the one call.
 * Outputs (DEVICE): out_tokens / out_parent int32[max_nodes] (entries [0, T)
 * written), out_T int32[1], out_info int32[3] = (matched n, 0 when none; hint
 * lanes used; all lanes used).  Stream-ordered.  Returns OOS_EINVAL on a NULL
 * or out-of-range argument, OOS_EWORKSPACE on a small or misaligned workspace. */
size_t oos_hint_workspace_bytes(int32_t bank_len);
int oos_hint_tree(const int32_t* bank, int32_t bank_len, int32_t eos, const int32_t* prefix, int32_t prefix_len,
                  const int32_t* native, const int32_t* native_len, int32_t n_native, int32_t native_stride,
                  int32_t max_lanes, int32_t depth, int32_t max_nodes, void* workspace, size_t ws_bytes,
                  int32_t* out_tokens, int32_t* out_parent, int32_t* out_T, int32_t* out_info, void* stream);

/* Target prefill: the step before tree verification, which fills the cache
 * with a prompt (the paper's targets start decoding from a prefilled request).
 *   kv            cache; slots [0, ctx_len) are read, slots [ctx_len,
 *                 ctx_len + n) receive the prompt's K/V.
 *   tokens        DEVICE int32[n], the prompt after the ctx_len cached positions.
 *   n             >= 1; any length that fits the cache: it runs as chains of at
 *                 most max_T tokens, each a tree pass of the verify kernels (a
 *                 chain's tree attention is causal attention).
 *   out_next_token  DEVICE int32[1] or NULL: the greedy next token after the
 *                 prompt (argmax of the last position's logits, Eq. 1).
 * Stream-ordered, no host synchronisation.  Returns OOS_EINVAL on NULL handle,
 * cache or tokens, n < 1 or ctx_len < 0; OOS_ECAPACITY when ctx_len + n exceeds
 * the cache; a token outside [0, vocab) is reported by oos_last_status
 * (OOS_ETREE), as for a tree. */
int oos_prefill(oos_model* m, const oos_kv_cache* kv, int32_t ctx_len, const int32_t* tokens, int32_t n,
                int32_t* out_next_token, void* stream);

/* Multi-step decoding on the device: the decoding loop of Section 2 ("The
 * ToolSpec decoding loop") with this library's verifier, n_rounds rounds with
 * no host round trip between them.  One round:
 *   1. the next tree from the hint bank, exactly as oos_hint_tree builds it,
 *      with the committed tokens as the prefix (their last token is the root),
 *      no native lanes, and max_nodes as the node budget;
 *   2. one verification of that tree (oos_tree_verify) at the committed cache
 *      length; the tree is padded to max_nodes nodes on the device, and the
 *      padding is never accepted;
 *   3. compaction of the accepted path (oos_kv_compact);
 *   4. the commit ("Verify and commit"): the accepted draft tokens and the
 *      bonus are appended to `committed` -- accepted_len tokens, the round's
 *      #MAT of Section 5 -- and the committed cache length grows by
 *      accepted_len (the root's K/V entered the cache; the bonus is the next
 *      root, its K/V written by the round that verifies it).
 * Arguments:
 *   kv             cache; slots [0, ctx_len) are committed.  Needs
 *                  ctx_len + n_rounds * max_nodes <= capacity.
 *   committed      DEVICE int32[committed_cap]: the committed tokens
 *                  [0, committed_len) (at least the root); the call appends.
 *                  Needs committed_len + n_rounds * max_nodes <= committed_cap.
 *   bank, bank_len, eos, max_lanes, depth   as oos_hint_tree (DEVICE bank).
 *   max_nodes      node budget of every tree, 1..max_T of the handle.
 *   out_mat        DEVICE int32[n_rounds]: accepted_len of every round.
 *   out_state      DEVICE int32[3]: after the call, the committed cache length,
 *                  the committed token count and the rounds run.
 *   workspace      DEVICE, >= oos_decode_workspace_bytes(bank_len), 256-byte
 *                  aligned; caller-owned scratch for the call.
 * Stream-ordered.  Host errors: OOS_EINVAL, OOS_ECAPACITY, OOS_EWORKSPACE,
 * OOS_ECUDA.  Device errors (a wait limit) go to oos_last_status; a round
 * whose verification failed commits nothing. */
size_t oos_decode_workspace_bytes(int32_t bank_len);
int oos_decode(oos_model* m, const oos_kv_cache* kv, int32_t ctx_len, int32_t* committed, int32_t committed_len,
               int32_t committed_cap, const int32_t* bank, int32_t bank_len, int32_t eos, int32_t max_lanes,
               int32_t depth, int32_t max_nodes, int32_t n_rounds, int32_t* out_mat, int32_t* out_state,
               void* workspace, size_t ws_bytes, void* stream);

/* One verification step (Eq. 1; "Verify and commit").
 *   kv            committed cache; slots [0, ctx_len) are read, slots
 *                 [ctx_len, ctx_len+T) are overwritten with the tree's K/V.
 *   ctx_len       committed positions already in the cache (>= 0).
 *   tree_tokens   DEVICE int32[T]: token of each node, node 0 = root.
 *   tree_parent   DEVICE int32[T]: parent of each node, parent[0] = -1.
 *   T             nodes, 1..max_T.
 * Outputs (DEVICE):
 *   out_accepted_len     int32[1]: nodes on the committed path, root included
 *                        (>= 1; the per-call "accepted tokens" of the paper's
 *                        #MAT metric), 0 on a device-detected error.
 *   out_accepted_nodes   int32[T]: node ids root-first; entries past len are -1.
 *   out_accepted_tokens  int32[T]: their tokens; entries past len are -1.
 *   out_bonus_token      int32[1]: the target's next token after the path.
 * The tree's K/V stay in slots ctx_len.. until oos_kv_compact. */
int oos_tree_verify(oos_model* m, const oos_kv_cache* kv, int32_t ctx_len,
                    const int32_t* tree_tokens, const int32_t* tree_parent, int32_t T,
                    int32_t* out_accepted_len, int32_t* out_accepted_nodes,
                    int32_t* out_accepted_tokens, int32_t* out_bonus_token, void* stream);

/* oos_tree_verify plus intermediate results for checking (DEVICE outputs):
 *   out_final_hidden  float[T, H]: output of the final RMSNorm per node (fp32)
 *   out_argmax        int32[T]:  the target's greedy token at every node
 *   out_top1/out_top2 float[T]:  largest and second-largest logit per node
 * Any of the four may be NULL. */
int oos_tree_verify_debug(oos_model* m, const oos_kv_cache* kv, int32_t ctx_len,
                          const int32_t* tree_tokens, const int32_t* tree_parent, int32_t T,
                          int32_t* out_accepted_len, int32_t* out_accepted_nodes,
                          int32_t* out_accepted_tokens, int32_t* out_bonus_token,
                          float* out_final_hidden, int32_t* out_argmax, float* out_top1,
                          float* out_top2, void* stream);

/* Commit the accepted path's K/V ("only states on the accepted target path
 * enter the committed KV cache").  For every layer and for K and V:
 * slot ctx_len + j <- slot ctx_len + accepted_nodes[j], j < *accepted_len, read
 * as a gather from the cache as it was before the call (sources never get
 * overwritten before they are read).  accepted_nodes / accepted_len are the
 * DEVICE outputs of oos_tree_verify (no host round trip); max_len is an upper
 * bound on *accepted_len (the T of that call).  The new committed length is
 * ctx_len + *accepted_len. */
int oos_kv_compact(oos_model* m, const oos_kv_cache* kv, int32_t ctx_len,
                   const int32_t* accepted_nodes, const int32_t* accepted_len, int32_t max_len,
                   void* stream);

/* Standalone greedy-acceptance walk over given argmax values (DEVICE in/out):
 * the same rule oos_tree_verify applies after its LM head.  Also validates the
 * tree; on a malformed tree *out_accepted_len = 0 and the call still returns
 * OOS_OK (the status is in *out_status: OOS_OK or OOS_ETREE). */
int oos_accept_walk(const int32_t* tree_tokens, const int32_t* tree_parent, const int32_t* argmax,
                    int32_t T, int32_t* out_accepted_len, int32_t* out_accepted_nodes,
                    int32_t* out_accepted_tokens, int32_t* out_bonus_token, int32_t* out_status,
                    void* stream);

/* Benchmarking aid: enqueue ONE weight-streaming kernel of the verify step
 * (with its fused epilogue), launched exactly as oos_tree_verify launches it,
 * on whatever activations the workspace holds.  stage: OOS_STAGE_O,
 * OOS_STAGE_GATE_UP, OOS_STAGE_DOWN (of layer `layer`) or OOS_STAGE_LM_HEAD
 * (layer ignored); T as in the last verify.  It writes only workspace scratch,
 * so the KV cache and the outputs of the last verify stay as they were, but
 * the workspace no longer holds that verify's intermediates.  OOS_STAGE_QKV
 * returns OOS_EINVAL for bf16 models: its epilogue writes the KV cache. */
#define OOS_STAGE_QKV 0
#define OOS_STAGE_O 1
#define OOS_STAGE_GATE_UP 2
#define OOS_STAGE_DOWN 3
#define OOS_STAGE_LM_HEAD 4
int oos_launch_stage(oos_model* m, int32_t layer, int32_t stage, int32_t T, void* stream);

/* Benchmarking aid: enqueue ONE tree-attention kernel of layer `layer`,
 * launched exactly as oos_tree_verify launches it, over cache positions
 * [0, ctx_len) of `kv` and the tree K/V in slots ctx_len..ctx_len+T-1 (as the
 * last verify with this ctx_len and T left them), with the workspace's q and
 * ancestor sets.  It reads the cache and writes only workspace scratch.
 * Errors as oos_tree_verify (EINVAL, ECAPACITY, ECUDA). */
int oos_launch_attention(oos_model* m, const oos_kv_cache* kv, int32_t layer, int32_t ctx_len, int32_t T,
                         void* stream);

/* LM-head greedy argmax that allocates nothing.  The paper has no counterpart:
 * this entry point exists for callers that cannot allocate device memory at
 * all -- code running inside someone else's CUDA-graph capture, under a memory
 * pool or allocator it does not own, or in a process whose allocator is locked
 * -- and so cannot provide the workspace oos_model_create needs.
 *   hidden      DEVICE float [T, hidden_dim]: final-RMSNorm rows (for example
 *               out_final_hidden of oos_tree_verify_debug).
 *   lm_head     DEVICE [vocab, hidden_dim], element type `dtype`.
 *   out_argmax  DEVICE int32 [T]: the v maximising hidden[t] . lm_head[v], the
 *               lowest such v on ties; out_top1 / out_top2 DEVICE float [T]:
 *               the largest and second-largest of those logits.
 * Scratch: a fixed 0.8 MB array in the library's device memory (allocated when
 * the library is loaded, held on every GPU that loads it until exit) holds the
 * per-block partial results; T must be <= 128, larger T returns OOS_EINVAL.
 * The kernel needs that array's device address, which a call made outside
 * stream capture looks up (cudaGetSymbolAddress) and caches for the device; a
 * call made while its stream is being captured uses the cached address.  So
 * make one uncaptured call on each device before any capture, and again after
 * a cudaDeviceReset.  Every call shares the array, so calls that may overlap
 * on the GPU (different streams, different host threads) race and must be
 * serialised by the caller.  CUDA cores only; a correctness and portability
 * path, not the fused tensor-core LM head of oos_tree_verify.  A row whose
 * logits contain NaN gets an unspecified argmax. */
int oos_lm_head_argmax_static(int32_t dtype, int32_t vocab, int32_t hidden_dim, const void* lm_head,
                              const float* hidden, int32_t T, int32_t* out_argmax, float* out_top1,
                              float* out_top2, void* stream);

/* Limit, in nanoseconds, of every pipeline wait inside this handle's kernels
 * (a TMA or tensor-core stage, a split-K partner, an attention split): a wait
 * that runs out sets OOS_ETIMEOUT in the status word, the kernel drains its
 * own copies and MMAs, frees its tensor memory and returns, and the rest of
 * the step returns early.  0 or a value above the default restores the
 * default of 2 s.  Meant for tests and diagnostics of the failure path (the
 * paper has no counterpart).  Applies to work enqueued on `stream` after the
 * call; synchronises `stream`. */
int oos_set_wait_limit(oos_model* m, uint64_t limit_ns, void* stream);

/* Synchronise `stream` and return the device status of the last verify on
 * this handle: OOS_OK, OOS_ETREE or OOS_ETIMEOUT (or OOS_ECUDA). */
int oos_last_status(oos_model* m, void* stream);

/* Static description of a status code. */
const char* oos_status_string(int code);

#ifdef __cplusplus
}
#endif

#endif /* OOS_H */
