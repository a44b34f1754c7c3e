// LM-head greedy argmax that allocates nothing (oos_lm_head_argmax_static).
//
// For callers that cannot allocate device memory at all -- code that runs
// inside a CUDA graph being captured by someone else, under a memory pool or
// allocator they do not own, or in a process whose allocator is locked -- this
// entry point needs no workspace: its per-block partial results live in a
// fixed file-scope device array that every call shares.
#include <mutex>

#include "common.cuh"
#include "internal.h"

namespace oos {

constexpr int kStaticBlocks = 512;   // vocabulary blocks per call (grid size)
constexpr int kStaticMaxT = 128;     // rows of `hidden` per call

struct StaticTop2 {
  float v1;
  int i1;
  float v2;
};

// Shared by every call on a device: [block][row] partial top-2 states, then the
// arrival counter (zero at load; the last block of a call sets it back to zero).
struct StaticScratch {
  StaticTop2 part[kStaticBlocks][kStaticMaxT];
  int arrived;
};
static __device__ __align__(256) StaticScratch g_argmax_scratch;

// Merge of two running top-2 states.  Order independent for finite logits (and
// infinities); a NaN logit compares false everywhere, so rows whose logits
// contain NaN get a layout-dependent result.
OOS_DEV StaticTop2 st_merge(StaticTop2 a, StaticTop2 b) {
  StaticTop2 r;
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

// Block b scans vocabulary rows [b*rows, (b+1)*rows): warp w takes rows
// w, w+4, ..., lanes stride over the hidden dimension; every row's logit for
// each of the T hidden rows updates that warp's running top-2.  The last block
// to finish merges all blocks' states, in block order.
template <typename E>
__global__ void __launch_bounds__(128) k_lm_argmax_static(const E* __restrict__ W, int V, int H, int rows_per_block,
                                                          const float* __restrict__ hidden, int T, StaticScratch* sc,
                                                          int32_t* out_argmax, float* out_top1, float* out_top2) {
  __shared__ StaticTop2 st[4][kStaticMaxT];
  __shared__ int s_last;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int t = lane; t < T; t += 32) st[warp][t] = StaticTop2{-INFINITY, 0x7fffffff, -INFINITY};
  __syncwarp();   // lane 0 below reads states the other lanes initialised
  const int r_begin = blockIdx.x * rows_per_block;
  const int r_end = min(V, r_begin + rows_per_block);
  for (int r = r_begin + warp; r < r_end; r += 4) {
    const E* w = W + (size_t)r * H;
    for (int t = 0; t < T; ++t) {
      const float* h = hidden + (size_t)t * H;
      float acc = 0.f;
      for (int k = lane; k < H; k += 32) acc += to_f32(w[k]) * h[k];
      acc = warp_sum(acc);
      if (lane == 0) st[warp][t] = st_merge(st[warp][t], StaticTop2{acc, r, -INFINITY});
    }
  }
  __syncthreads();
  for (int t = threadIdx.x; t < T; t += blockDim.x) {
    StaticTop2 r = st[0][t];
    for (int w = 1; w < 4; ++w) r = st_merge(r, st[w][t]);
    sc->part[blockIdx.x][t] = r;
  }
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) {
    const int old = atomicAdd(&sc->arrived, 1);
    s_last = old == (int)gridDim.x - 1;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  for (int t = threadIdx.x; t < T; t += blockDim.x) {
    StaticTop2 r{-INFINITY, 0x7fffffff, -INFINITY};
    for (int b = 0; b < (int)gridDim.x; ++b) {
      const StaticTop2 p{__ldcg(&sc->part[b][t].v1), __ldcg(&sc->part[b][t].i1), __ldcg(&sc->part[b][t].v2)};
      r = st_merge(r, p);
    }
    out_argmax[t] = r.i1;
    out_top1[t] = r.v1;
    out_top2[t] = r.v2;
  }
  if (threadIdx.x == 0) sc->arrived = 0;   // the next call starts from zero
}

// Device address of the scratch array.  In host code g_argmax_scratch names a
// host-side stand-in, not device memory, so the kernel is given the address
// cudaGetSymbolAddress returns for the current device.  Outside stream
// capture it is looked up on every call (cheap, and right again after a
// cudaDeviceReset reloads the module); a call made while its stream is being
// captured uses the address cached by the last uncaptured call on the device.
static std::mutex g_scratch_mu;
static StaticScratch* g_scratch_ptr[64];

static StaticScratch* scratch_for_current_device(cudaStream_t st) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(st, &cs) != cudaSuccess) return nullptr;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (cs == cudaStreamCaptureStatusNone) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_argmax_scratch) != cudaSuccess) return nullptr;
    g_scratch_ptr[dev] = static_cast<StaticScratch*>(p);
  }
  return g_scratch_ptr[dev];
}

}  // namespace oos

using namespace oos;

extern "C" int oos_lm_head_argmax_static(int32_t dtype, int32_t vocab, int32_t hidden_dim, const void* lm_head,
                                         const float* hidden, int32_t T, int32_t* out_argmax, float* out_top1,
                                         float* out_top2, void* stream) {
  if (!lm_head || !hidden || !out_argmax || !out_top1 || !out_top2) return OOS_EINVAL;
  if (dtype != OOS_DTYPE_F32 && dtype != OOS_DTYPE_BF16) return OOS_EINVAL;
  if (vocab < 1 || hidden_dim < 1) return OOS_EINVAL;
  if (T < 1 || T > kStaticMaxT) return OOS_EINVAL;   // the scratch array holds kStaticMaxT rows
  cudaStream_t st = (cudaStream_t)stream;
  StaticScratch* sc = scratch_for_current_device(st);
  if (!sc) return OOS_ECUDA;
  const int blocks = vocab < kStaticBlocks ? vocab : kStaticBlocks;
  const int rows = (vocab + blocks - 1) / blocks;
  if (dtype == OOS_DTYPE_BF16)
    k_lm_argmax_static<__nv_bfloat16><<<blocks, 128, 0, st>>>((const __nv_bfloat16*)lm_head, vocab, hidden_dim, rows,
                                                             hidden, T, sc, out_argmax, out_top1, out_top2);
  else
    k_lm_argmax_static<float><<<blocks, 128, 0, st>>>((const float*)lm_head, vocab, hidden_dim, rows, hidden, T, sc,
                                                      out_argmax, out_top1, out_top2);
  return cudaGetLastError() == cudaSuccess ? OOS_OK : OOS_ECUDA;
}
