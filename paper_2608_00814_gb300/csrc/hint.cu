// Hint-bank candidate step: the next verification tree from the request's
// hint bank (Section 4, "Suffix matching" and "Candidate boundary").
//
// The committed prefix y is matched against the bank (tokenised views joined
// by EOS): for n = 7 down to 1 the length-n suffix of y is searched, and the
// tokens after each occurrence become candidate lanes, ahead of the native
// lanes, under a lane budget; the lanes are packed into a prefix tree rooted
// at y's last token.  An occurrence counts only when a non-EOS token follows
// it; the longest n with any counted occurrence is used; lanes are taken in
// bank order, cut at the lane depth or before an EOS; a lane counts towards
// the budget only when it creates a node.
//
// k_hint_match: for every bank position the longest n whose suffix ends
// there (0 when nothing, or EOS, follows), as one byte; a warp per 256-position
// chunk, 8 positions per lane; the maximum of each chunk and of each run of 256
// chunks (a "span") is kept too, and the warp maxima give the n of the call.  k_hint_pack: one block descends the two summaries in bank order --
// spans, then their chunks, then positions, 256 at a time, each level's hits
// gathered in order by warp ballots -- so only spans and chunks that hold an
// occurrence are read, and warp 0 inserts each lane into the tree held in
// shared memory: a lane token looks for an existing child with one ballot over
// the nodes.
#include <stdint.h>

#include "common.cuh"
#include "internal.h"

namespace oos {

constexpr int kHintMaxN = 7;        // longest suffix tried
constexpr int kHintThreads = 256;   // threads of both kernels

// prefix_len_dev: the prefix length in device memory (the decode loop's
// committed length), or nullptr to use prefix_len.  Each warp takes one
// 256-position chunk at a time (grid-stride over chunks), each lane 8
// consecutive positions: the lane reads bank[p0 - 8, p0 + 16) (vector loads
// when the bank is 16-byte aligned), computes the 8 match lengths, stores
// them as 8 bytes, and the chunk maximum is a warp reduction -- no block
// barrier.  vec: the bank address is 16-byte aligned.
__global__ void __launch_bounds__(kHintThreads) k_hint_match(const int32_t* __restrict__ bank, int N, int eos,
                                                             const int32_t* __restrict__ prefix, int prefix_len,
                                                             const int32_t* __restrict__ prefix_len_dev, int vec,
                                                             uint8_t* __restrict__ mlen, uint8_t* __restrict__ cmax,
                                                             int* __restrict__ smax, int* __restrict__ best) {
  __shared__ int suf[kHintMaxN];
  pdl_wait();   // the committed tokens and their count may come from the previous kernel
  pdl_trigger();
  if (prefix_len_dev) prefix_len = *prefix_len_dev;
  const int nmax = prefix_len < kHintMaxN ? prefix_len : kHintMaxN;
  // suf[j] is the token j places before y's last token
  if (threadIdx.x < nmax) suf[threadIdx.x] = prefix[prefix_len - 1 - threadIdx.x];
  __syncthreads();
  int sfx[kHintMaxN];
#pragma unroll
  for (int j = 0; j < kHintMaxN; ++j) sfx[j] = j < nmax ? suf[j] : 0;
  const int lane = threadIdx.x & 31;
  const long long n_chunks = ((long long)N + kHintThreads - 1) / kHintThreads;
  const long long n_warps = (long long)gridDim.x * (kHintThreads / 32);
  int wbest = 0;
  for (long long c = (long long)blockIdx.x * (kHintThreads / 32) + (threadIdx.x >> 5); c < n_chunks; c += n_warps) {
    const long long p0 = c * kHintThreads + lane * 8;
    int w[24];   // bank[p0 - 8 + i]; positions outside [0, N) are never compared
    if (vec && p0 >= 8 && p0 + 16 <= N) {
      const int4* src = reinterpret_cast<const int4*>(bank + p0 - 8);
#pragma unroll
      for (int q = 0; q < 6; ++q) {
        const int4 v = __ldcs(src + q);
        w[4 * q] = v.x;
        w[4 * q + 1] = v.y;
        w[4 * q + 2] = v.z;
        w[4 * q + 3] = v.w;
      }
    } else {
#pragma unroll
      for (int i = 0; i < 24; ++i) {
        const long long q = p0 - 8 + i;
        w[i] = (q >= 0 && q < N) ? bank[q] : 0;
      }
    }
    uint32_t packed[2] = {0u, 0u};
    int lmax = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const long long p = p0 + i;
      int m = 0;
      // the next bank token must exist and not be EOS
      if (p + 1 < N && w[9 + i] != eos) {
#pragma unroll
        for (int j = 0; j < kHintMaxN; ++j) {
          if (m < j || j >= nmax || p - j < 0 || w[8 + i - j] != sfx[j]) break;
          m = j + 1;
        }
      }
      packed[i >> 2] |= (uint32_t)m << (8 * (i & 3));
      lmax = m > lmax ? m : lmax;
    }
    if (p0 + 8 <= N) {
      *reinterpret_cast<uint2*>(mlen + p0) = make_uint2(packed[0], packed[1]);
    } else {
      for (int i = 0; i < 8 && p0 + i < N; ++i) mlen[p0 + i] = (uint8_t)((packed[i >> 2] >> (8 * (i & 3))) & 255u);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) lmax = max(lmax, __shfl_xor_sync(0xffffffffu, lmax, o));
    if (lane == 0) {
      cmax[c] = (uint8_t)lmax;
      if (lmax > 0) atomicMax(&smax[c / kHintThreads], lmax);
    }
    wbest = max(wbest, lmax);
  }
  if (lane == 0 && wbest > 0) atomicMax(best, wbest);
}

// Whole block: the values of the threads whose `has` is set, in thread order,
// into out[0..count); returns count (the same in every thread).  Two block
// barriers; every thread of the block must call it.
OOS_DEV int ordered_select(bool has, int32_t value, int32_t* out, int* s_wcnt, int* s_cnt) {
  const int warp = threadIdx.x >> 5, lane_id = threadIdx.x & 31;
  const unsigned bal = __ballot_sync(0xffffffffu, has);
  if (lane_id == 0) s_wcnt[warp] = __popc(bal);
  __syncthreads();
  if (has) {
    int off = __popc(bal & ((1u << lane_id) - 1u));
    for (int w = 0; w < warp; ++w) off += s_wcnt[w];
    out[off] = value;
  }
  if (threadIdx.x == 0) {
    int k = 0;
    for (int w = 0; w < kHintThreads / 32; ++w) k += s_wcnt[w];
    *s_cnt = k;
  }
  __syncthreads();
  return *s_cnt;
}

// Insert one lane into the tree (warp 0, all lanes of the warp together).
// Returns whether a node was created.  The caller stops when the lane or
// node budget is spent.
OOS_DEV bool hint_insert(int32_t* s_tok, int32_t* s_par, int& T, int max_nodes, const int32_t* lane, int len) {
  const int lane_id = threadIdx.x & 31;
  int cur = 0;
  bool created = false;
  for (int j = 0; j < len; ++j) {
    const int t = lane[j];
    // the child of cur with token t, if any (nodes are distinct per (parent, token))
    int found = -1;
    for (int base = 1; base < T && found < 0; base += 32) {
      const int i = base + lane_id;
      const unsigned hit = __ballot_sync(0xffffffffu, i < T && s_par[i] == cur && s_tok[i] == t);
      if (hit) found = base + __ffs(hit) - 1;
    }
    if (found >= 0) {
      cur = found;
      continue;
    }
    if (T >= max_nodes) break;
    if (lane_id == 0) {
      s_tok[T] = t;
      s_par[T] = cur;
    }
    __syncwarp();
    cur = T;
    ++T;
    created = true;
  }
  return created;
}

__global__ void __launch_bounds__(kHintThreads) k_hint_pack(const int32_t* __restrict__ bank, int N, int eos,
                                                            const int32_t* __restrict__ prefix, int prefix_len,
                                                            const uint8_t* __restrict__ mlen,
                                                            const uint8_t* __restrict__ cmax,
                                                            const int* __restrict__ smax,
                                                            const int* __restrict__ best,
                                                            const int32_t* __restrict__ native,
                                                            const int32_t* __restrict__ native_len, int n_native,
                                                            int native_stride, int max_lanes, int depth,
                                                            int max_nodes, const int32_t* __restrict__ prefix_len_dev,
                                                            int pad_to, int32_t* out_tok, int32_t* out_par,
                                                            int32_t* out_T, int32_t* out_info) {
  __shared__ int32_t s_tok[kMaxT], s_par[kMaxT];
  __shared__ int32_t s_pos[kHintThreads];     // occurrences in the chunk being visited, in bank order
  __shared__ int32_t s_chunk[kHintThreads];   // the span's chunks holding an occurrence, in order
  __shared__ int32_t s_span[kHintThreads];    // this round's spans holding an occurrence, in order
  __shared__ int32_t s_lane[kMaxT];           // the lane being inserted
  __shared__ int s_wcnt[kHintThreads / 32];
  __shared__ int s_n, s_nc, s_ns, s_done;
  const int warp = threadIdx.x >> 5, lane_id = threadIdx.x & 31;
  pdl_wait();   // the match kernel's results
  pdl_trigger();
  const int n = *best;
  if (prefix_len_dev) prefix_len = *prefix_len_dev;
  int T = 1, lanes = 0, hint_lanes = 0;       // warp 0's copies are the authoritative ones
  if (threadIdx.x == 0) {
    s_tok[0] = prefix[prefix_len - 1];
    s_par[0] = -1;
    s_done = (max_lanes <= 0 || max_nodes <= 1) ? 1 : 0;
  }
  __syncthreads();
  // hint lanes: occurrences of the length-n suffix (match length >= n), bank order
  const long long n_chunks = ((long long)N + kHintThreads - 1) / kHintThreads;
  const long long n_spans = (n_chunks + kHintThreads - 1) / kHintThreads;
  for (long long sb = 0; n > 0 && sb < n_spans; sb += kHintThreads) {
    if (s_done) break;
    const long long sp = sb + threadIdx.x;
    const int ns = ordered_select(sp < n_spans && smax[sp] >= n, (int32_t)sp, s_span, s_wcnt, &s_ns);
    for (int si = 0; si < ns; ++si) {
      if (s_done) break;
      const long long c = (long long)s_span[si] * kHintThreads + threadIdx.x;
      const int nc = ordered_select(c < n_chunks && cmax[c] >= n, (int32_t)c, s_chunk, s_wcnt, &s_nc);
      // visit the chunks: their occurrences in order, then warp 0 inserts their lanes
      for (int ci = 0; ci < nc; ++ci) {
        if (s_done) break;
        const long long p = (long long)s_chunk[ci] * kHintThreads + threadIdx.x;
        const int np = ordered_select(p < N && mlen[p] >= n, (int32_t)p, s_pos, s_wcnt, &s_n);
        if (warp == 0) {
          for (int k = 0; k < np; ++k) {
            if (lanes >= max_lanes || T >= max_nodes) break;
            // lane: up to depth tokens after the occurrence, stopping before an EOS
            const long long q0 = (long long)s_pos[k] + 1;
            int len = 0;
            for (int j = 0; j < depth; ++j) {
              const long long q = q0 + j;
              if (q >= N) break;
              const int t = bank[q];
              if (t == eos) break;
              if (lane_id == 0) s_lane[j] = t;
              ++len;
            }
            __syncwarp();
            if (hint_insert(s_tok, s_par, T, max_nodes, s_lane, len)) {
              ++lanes;
              ++hint_lanes;
            }
            __syncwarp();
          }
          if (lane_id == 0 && (lanes >= max_lanes || T >= max_nodes)) s_done = 1;
        }
        __syncthreads();
      }
    }
  }
  // native lanes fill what the budgets leave
  if (warp == 0) {
    for (int i = 0; i < n_native; ++i) {
      if (lanes >= max_lanes || T >= max_nodes) break;
      int len = native_len[i];
      len = len < depth ? len : depth;
      len = len < native_stride ? len : native_stride;
      len = len < 0 ? 0 : len;
      for (int j = lane_id; j < len; j += 32) s_lane[j] = native[(size_t)i * native_stride + j];
      __syncwarp();
      if (hint_insert(s_tok, s_par, T, max_nodes, s_lane, len)) ++lanes;
      __syncwarp();
    }
    for (int i = lane_id; i < T; i += 32) {
      out_tok[i] = s_tok[i];
      out_par[i] = s_par[i];
    }
    // padding up to a fixed node count (the decode loop verifies a fixed T):
    // leaves under the root carrying the root's token; the verifier is told
    // the real node count and never accepts them
    for (int i = T + lane_id; i < pad_to; i += 32) {
      out_tok[i] = s_tok[0];
      out_par[i] = 0;
    }
    if (lane_id == 0) {
      *out_T = T;
      out_info[0] = n;
      out_info[1] = hint_lanes;
      out_info[2] = lanes;
    }
  }
}

// workspace: [best | pad to 256][mlen: one byte per position, padded to 256]
//            [cmax: one byte per chunk, padded to 256][smax: one int per span]
// Workspace: the call's n (best) and the span maxima first, so that one
// zeroing copy covers both; then one match byte per position and the chunk maxima.
static size_t hint_head_bytes(size_t spans) { return (4 + spans * 4 + 255) / 256 * 256; }

size_t hint_workspace_bytes(long long bank_len) {
  const size_t chunks = (size_t)((bank_len + kHintThreads - 1) / kHintThreads);
  const size_t spans = (chunks + kHintThreads - 1) / kHintThreads;
  return hint_head_bytes(spans) + chunks * kHintThreads + spans * kHintThreads;
}

cudaError_t launch_hint_tree(const int32_t* bank, int N, int eos, const int32_t* prefix, int prefix_len,
                             const int32_t* prefix_len_dev, const int32_t* native, const int32_t* native_len,
                             int n_native, int native_stride, int max_lanes, int depth, int max_nodes, int pad_to,
                             void* ws, int32_t* out_tok, int32_t* out_par, int32_t* out_T, int32_t* out_info,
                             cudaStream_t st) {
  const long long n_chunks = ((long long)N + kHintThreads - 1) / kHintThreads;
  const long long n_spans = (n_chunks + kHintThreads - 1) / kHintThreads;
  int* best = (int*)ws;
  int* smax = best + 1;
  uint8_t* mlen = (uint8_t*)ws + hint_head_bytes((size_t)n_spans);
  uint8_t* cmax = mlen + n_chunks * kHintThreads;
  cudaError_t e = cudaMemsetAsync(best, 0, (size_t)(1 + n_spans) * sizeof(int), st);
  if (e != cudaSuccess) return e;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  // one warp per 256-position chunk; enough blocks for every SM to hold several
  const long long want = (n_chunks + kHintThreads / 32 - 1) / (kHintThreads / 32);
  const int grid = (int)(want < (long long)sms * 8 ? want : (long long)sms * 8);
  const int vec = ((uintptr_t)bank & 15) == 0 ? 1 : 0;
  // the packing block launches while the match kernel runs (programmatic
  // dependent launch) and waits for it before reading its results
  e = launch(true, k_hint_match, dim3(grid), dim3(kHintThreads), 0, st, bank, N, eos, prefix, prefix_len,
             prefix_len_dev, vec, mlen, cmax, smax, best);
  if (e != cudaSuccess) return e;
  return launch(true, k_hint_pack, dim3(1), dim3(kHintThreads), 0, st, bank, N, eos, prefix, prefix_len,
                (const uint8_t*)mlen, (const uint8_t*)cmax, (const int*)smax, (const int*)best, native, native_len,
                n_native, native_stride, max_lanes, depth, max_nodes, prefix_len_dev, pad_to, out_tok, out_par, out_T,
                out_info);
}

}  // namespace oos

using namespace oos;

extern "C" {

size_t oos_hint_workspace_bytes(int32_t bank_len) { return bank_len < 1 ? 0 : hint_workspace_bytes(bank_len); }

int oos_hint_tree(const int32_t* bank, int32_t bank_len, int32_t eos, const int32_t* prefix, int32_t prefix_len,
                  const int32_t* native, const int32_t* native_len, int32_t n_native, int32_t native_stride,
                  int32_t max_lanes, int32_t depth, int32_t max_nodes, void* workspace, size_t ws_bytes,
                  int32_t* out_tokens, int32_t* out_parent, int32_t* out_T, int32_t* out_info, void* stream) {
  if (!bank || bank_len < 1 || !prefix || prefix_len < 1 || n_native < 0 || max_lanes < 0) return OOS_EINVAL;
  if (n_native > 0 && (!native || !native_len || native_stride < 1)) return OOS_EINVAL;
  if (depth < 1 || depth > kMaxT || max_nodes < 1 || max_nodes > kMaxT) return OOS_EINVAL;
  if (!out_tokens || !out_parent || !out_T || !out_info) return OOS_EINVAL;
  if (!workspace || ((uintptr_t)workspace & 255) || ws_bytes < hint_workspace_bytes(bank_len)) return OOS_EWORKSPACE;
  return launch_hint_tree(bank, bank_len, eos, prefix, prefix_len, nullptr, native, native_len, n_native,
                          native_stride, max_lanes, depth, max_nodes, 0, workspace, out_tokens, out_parent, out_T,
                          out_info, (cudaStream_t)stream) == cudaSuccess
             ? OOS_OK
             : OOS_ECUDA;
}

}  // extern "C"
