// Tree attention of the verify step.
//
// Node i, query head h (kv head g = h / (nq/nkv)) attends to the committed
// cache positions [0, ctx) and to the tree slots ctx + a for every ancestor a
// of i (itself included): softmax(q k / sqrt(d)) v.
//
// bf16 path: split-K over the cache (flash-decoding).  A block owns 64 query
// rows of one kv head -- the (node, q-head) pairs of the group, so GQA reuses
// every K/V tile for nq/nkv heads -- and one range of cache keys; the last
// split also takes the tree tail, masked with the 128-bit ancestor sets.  K/V
// tiles are staged in shared memory by a 3-deep cp.async ring; scores and P.V
// run on the tensor cores (mma.sync m16n8k16, fp32 accumulate) with an online
// softmax in fp32.  The last split of a row block to finish merges all splits
// by log-sum-exp (fixed split order) and writes the hi/lo bf16 GEMM input.
//
// fp32 path: one block per (node, head), CUDA cores (small models only).
#include <math.h>
#include <stdlib.h>

#include "common.cuh"
#include "internal.h"

namespace oos {

constexpr int kAttnRows = 64;     // query rows per block (4 warps x 16)
constexpr int kAttnKeys = 64;     // keys per tile
constexpr int kAttnD = 128;       // head dim of the bf16 path
constexpr int kAttnLd = kAttnD + 8;   // padded smem row (272 bytes): conflict-free ldmatrix
constexpr int kAttnStages = 3;        // cp.async ring of K/V tiles
constexpr int kAttnStageElems = 2 * kAttnKeys * kAttnLd;   // K tile then V tile
constexpr int kAttnSmem = kAttnStages * kAttnStageElems * 2;

struct AttnArgs {
  const __nv_bfloat16* q;   // [T][nq][d]
  const __nv_bfloat16* kc;  // [cap][nkv][d]
  const __nv_bfloat16* vc;
  const unsigned long long* anc;
  int T, nq, nkv, group, ctx;
  int splits, cache_blocks, row_blocks;
  float scale_log2;         // log2(e) / sqrt(d)
  float* o_part;            // [split][T*nq][d]
  float* ml_part;           // [split][T*nq][2]
  int* cnt;                 // [nkv * row_blocks] split arrival counters
  __nv_bfloat16* out;       // [T][nq*d] hi rows, lo rows at out_lo_off
  size_t out_lo_off;
};

OOS_DEV void cp_async16(void* smem, const void* gmem, bool valid) {
  const int n = valid ? 16 : 0;
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_addr(smem)), "l"(gmem), "r"(n) : "memory");
}
OOS_DEV void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
OOS_DEV void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

OOS_DEV void ldsm_x4(uint32_t (&r)[4], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(smem_addr(p)));
}
OOS_DEV void ldsm_x4_t(uint32_t (&r)[4], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(smem_addr(p)));
}
// pure register operation: not volatile, so the compiler may interleave
// independent MMAs with loads and each other
OOS_DEV void mma_bf16(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
OOS_DEV uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// stage 64 keys (cache positions or tree slots) of kv head g into smem
OOS_DEV void load_kv_tile(__nv_bfloat16* ks, __nv_bfloat16* vs, const AttnArgs& a, int g, int key0, int key_end) {
  for (int c = threadIdx.x; c < kAttnKeys * (kAttnD / 8); c += blockDim.x) {
    const int r = c >> 4, col = (c & 15) * 8;
    const int key = key0 + r;
    const bool valid = key < key_end;
    const size_t off = ((size_t)(valid ? key : key0) * a.nkv + g) * kAttnD + col;
    cp_async16(ks + r * kAttnLd + col, a.kc + off, valid);
    cp_async16(vs + r * kAttnLd + col, a.vc + off, valid);
  }
}

__global__ void __launch_bounds__(128) k_attn_tc(AttnArgs a) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  __nv_bfloat16* ring = reinterpret_cast<__nv_bfloat16*>(smem_raw);   // [stage][K | V][64][ld]
  __shared__ int s_last;
  __shared__ float s_w[kAttnRows][kMaxAttnSplits];   // merge weights (last split only)
  pdl_trigger();
  pdl_wait();
  const int rb = blockIdx.x, g = blockIdx.y, split = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int R = a.T * a.group;

  // key tiles of this block: cache blocks [cb0, cb1), then (last split) the tree tail
  const int cb0 = (int)((long long)split * a.cache_blocks / a.splits);
  const int cb1 = (int)((long long)(split + 1) * a.cache_blocks / a.splits);
  const int tree_tiles = (split == a.splits - 1) ? (a.T + kAttnKeys - 1) / kAttnKeys : 0;
  const int n_tiles = (cb1 - cb0) + tree_tiles;
  auto tile_keys = [&](int ti, int& key0, int& key_end, bool& tree) {
    if (ti < cb1 - cb0) {
      key0 = (cb0 + ti) * kAttnKeys;
      key_end = min(a.ctx, key0 + kAttnKeys);
      tree = false;
    } else {
      const int tt = ti - (cb1 - cb0);
      key0 = a.ctx + tt * kAttnKeys;
      key_end = a.ctx + a.T;
      tree = true;
    }
  };
  auto stage_k = [&](int s) { return ring + s * kAttnStageElems; };
  auto stage_v = [&](int s) { return ring + s * kAttnStageElems + kAttnKeys * kAttnLd; };
  auto issue = [&](int ti) {
    if (ti < n_tiles) {
      int k0, ke;
      bool tr;
      tile_keys(ti, k0, ke, tr);
      load_kv_tile(stage_k(ti % kAttnStages), stage_v(ti % kAttnStages), a, g, k0, ke);
    }
    cp_async_commit();
  };

  // Q rows (row r -> node r / group, head g*group + r % group), staged through
  // the last ring slot, then kept in registers as mma A fragments
  {
    __nv_bfloat16* Qs = stage_k(kAttnStages - 1);
    for (int c = threadIdx.x; c < kAttnRows * (kAttnD / 8); c += blockDim.x) {
      const int r = c >> 4, col = (c & 15) * 8;
      const int row = rb * kAttnRows + r;
      const bool valid = row < R;
      const int node = valid ? row / a.group : 0, hq = g * a.group + (valid ? row % a.group : 0);
      cp_async16(Qs + r * kAttnLd + col, a.q + ((size_t)node * a.nq + hq) * kAttnD + col, valid);
    }
    cp_async_commit();
    cp_async_wait<0>();
    __syncthreads();
  }
  uint32_t qf[8][4];
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
    const int row = warp * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
    const int col = ks * 16 + (lane >> 4) * 8;
    ldsm_x4(qf[ks], stage_k(kAttnStages - 1) + row * kAttnLd + col);
  }
  __syncthreads();
  issue(0);
  issue(1);

  // per-thread rows: r_lo = warp*16 + lane/4, r_hi = r_lo + 8
  const int r_lo = rb * kAttnRows + warp * 16 + (lane >> 2);
  const int r_hi = r_lo + 8;
  const int node_lo = min(r_lo, R - 1) / a.group, node_hi = min(r_hi, R - 1) / a.group;
  const unsigned long long anc_lo0 = a.anc[2 * node_lo], anc_lo1 = a.anc[2 * node_lo + 1];
  const unsigned long long anc_hi0 = a.anc[2 * node_hi], anc_hi1 = a.anc[2 * node_hi + 1];

  float o[16][4];
#pragma unroll
  for (int n = 0; n < 16; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;
  float m_lo = -INFINITY, m_hi = -INFINITY, l_lo = 0.f, l_hi = 0.f;

  for (int ti = 0; ti < n_tiles; ++ti) {
    issue(ti + 2);
    cp_async_wait<2>();
    __syncthreads();
    const __nv_bfloat16* kt = stage_k(ti % kAttnStages);
    const __nv_bfloat16* vt = stage_v(ti % kAttnStages);
    int key0, key_end;
    bool tree;
    tile_keys(ti, key0, key_end, tree);

    // S = Q K^T  (16 rows x 64 keys per warp); k-steps outer, key groups inner,
    // so consecutive MMAs write different accumulators
    float s[8][4];
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
#pragma unroll
    for (int ks = 0; ks < 8; ks += 2) {
      uint32_t b[8][4];
#pragma unroll
      for (int nt = 0; nt < 8; ++nt)
        ldsm_x4(b[nt], kt + (nt * 8 + (lane & 7)) * kAttnLd + ks * 16 + (lane >> 3) * 8);
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) mma_bf16(s[nt], qf[ks], b[nt][0], b[nt][1]);
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) mma_bf16(s[nt], qf[ks + 1], b[nt][2], b[nt][3]);
    }
    // scale (+ mask on the tree tail and a partial last cache tile), tile row maxima
    float tmax_lo = -INFINITY, tmax_hi = -INFINITY;
    if (tree || key_end < key0 + kAttnKeys) {
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int key = key0 + nt * 8 + (lane & 3) * 2 + (e & 1);
          bool valid = key < key_end;
          if (tree && valid) {
            const int j = key - a.ctx;
            const unsigned long long w0 = (e < 2) ? anc_lo0 : anc_hi0;
            const unsigned long long w1 = (e < 2) ? anc_lo1 : anc_hi1;
            valid = ((j < 64 ? (w0 >> j) : (w1 >> (j - 64))) & 1ull) != 0;
          }
          const float v = valid ? s[nt][e] * a.scale_log2 : -INFINITY;
          s[nt][e] = v;
          if (e < 2) tmax_lo = fmaxf(tmax_lo, v); else tmax_hi = fmaxf(tmax_hi, v);
        }
      }
    } else {
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
        for (int e = 0; e < 4; ++e) s[nt][e] *= a.scale_log2;
        tmax_lo = fmaxf(tmax_lo, fmaxf(s[nt][0], s[nt][1]));
        tmax_hi = fmaxf(tmax_hi, fmaxf(s[nt][2], s[nt][3]));
      }
    }
#pragma unroll
    for (int off = 1; off <= 2; off <<= 1) {
      tmax_lo = fmaxf(tmax_lo, __shfl_xor_sync(0xffffffffu, tmax_lo, off));
      tmax_hi = fmaxf(tmax_hi, __shfl_xor_sync(0xffffffffu, tmax_hi, off));
    }
    const float mn_lo = fmaxf(m_lo, tmax_lo), mn_hi = fmaxf(m_hi, tmax_hi);
    const float base_lo = mn_lo == -INFINITY ? 0.f : mn_lo;
    const float base_hi = mn_hi == -INFINITY ? 0.f : mn_hi;
    const float corr_lo = exp2f(m_lo - base_lo), corr_hi = exp2f(m_hi - base_hi);
    m_lo = mn_lo;
    m_hi = mn_hi;
    float sum_lo = 0.f, sum_hi = 0.f;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      s[nt][0] = exp2f(s[nt][0] - base_lo);
      s[nt][1] = exp2f(s[nt][1] - base_lo);
      s[nt][2] = exp2f(s[nt][2] - base_hi);
      s[nt][3] = exp2f(s[nt][3] - base_hi);
      sum_lo += s[nt][0] + s[nt][1];
      sum_hi += s[nt][2] + s[nt][3];
    }
    l_lo = l_lo * corr_lo + sum_lo;
    l_hi = l_hi * corr_hi + sum_hi;
#pragma unroll
    for (int n = 0; n < 16; ++n) {
      o[n][0] *= corr_lo;
      o[n][1] *= corr_lo;
      o[n][2] *= corr_hi;
      o[n][3] *= corr_hi;
    }
    // O += P V
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      uint32_t pa[4];
      pa[0] = pack_bf16(s[2 * kk][0], s[2 * kk][1]);
      pa[1] = pack_bf16(s[2 * kk][2], s[2 * kk][3]);
      pa[2] = pack_bf16(s[2 * kk + 1][0], s[2 * kk + 1][1]);
      pa[3] = pack_bf16(s[2 * kk + 1][2], s[2 * kk + 1][3]);
      uint32_t b[8][4];
      const int mi = lane >> 3;
#pragma unroll
      for (int n2 = 0; n2 < 16; n2 += 2)
        ldsm_x4_t(b[n2 / 2], vt + (kk * 16 + (mi & 1) * 8 + (lane & 7)) * kAttnLd + (n2 + (mi >> 1)) * 8);
#pragma unroll
      for (int n2 = 0; n2 < 16; n2 += 2) {
        mma_bf16(o[n2], pa, b[n2 / 2][0], b[n2 / 2][1]);
        mma_bf16(o[n2 + 1], pa, b[n2 / 2][2], b[n2 / 2][3]);
      }
    }
    __syncthreads();
  }
  cp_async_wait<0>();

  // quad sums of l, then this split's unnormalised O and (m, l)
#pragma unroll
  for (int off = 1; off <= 2; off <<= 1) {
    l_lo += __shfl_xor_sync(0xffffffffu, l_lo, off);
    l_hi += __shfl_xor_sync(0xffffffffu, l_hi, off);
  }
  const size_t rows_total = (size_t)a.T * a.nq;
#pragma unroll
  for (int half = 0; half < 2; ++half) {
    const int r = half ? r_hi : r_lo;
    if (r >= R) continue;
    const int node = r / a.group, hq = g * a.group + r % a.group;
    const size_t grow = (size_t)node * a.nq + hq;
    float* dst = a.o_part + ((size_t)split * rows_total + grow) * kAttnD;
#pragma unroll
    for (int n = 0; n < 16; ++n) {
      const int col = n * 8 + (lane & 3) * 2;
      *reinterpret_cast<float2*>(dst + col) = half ? make_float2(o[n][2], o[n][3]) : make_float2(o[n][0], o[n][1]);
    }
    if ((lane & 3) == 0) {
      float* ml = a.ml_part + ((size_t)split * rows_total + grow) * 2;
      ml[0] = half ? m_hi : m_lo;
      ml[1] = half ? l_hi : l_lo;
    }
  }

  // the last split of this (row block, kv head) to finish merges all splits:
  // log-sum-exp weights in base 2, summed in split order
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) {
    const int ci = g * a.row_blocks + rb;
    const int old = atomicAdd(&a.cnt[ci], 1);
    s_last = old == a.splits - 1;
    if (s_last) a.cnt[ci] = 0;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  // per-row split weights w_s = 2^(m_s - M) / sum_s 2^(m_s - M) l_s
  if (threadIdx.x < kAttnRows) {
    const int r = rb * kAttnRows + threadIdx.x;
    if (r < R) {
      const size_t grow = (size_t)(r / a.group) * a.nq + g * a.group + r % a.group;
      float ms[kMaxAttnSplits], ls[kMaxAttnSplits];
      float M = -INFINITY;
#pragma unroll
      for (int sp = 0; sp < kMaxAttnSplits; ++sp) {
        if (sp < a.splits) {
          const float2 v = __ldcg(reinterpret_cast<const float2*>(a.ml_part + ((size_t)sp * rows_total + grow) * 2));
          ms[sp] = v.x;
          ls[sp] = v.y;
          M = fmaxf(M, v.x);
        }
      }
      float den = 0.f;
#pragma unroll
      for (int sp = 0; sp < kMaxAttnSplits; ++sp) {
        if (sp < a.splits) {
          const float wgt = ms[sp] == -INFINITY ? 0.f : exp2f(ms[sp] - M);
          ms[sp] = wgt;
          den += wgt * ls[sp];
        }
      }
#pragma unroll
      for (int sp = 0; sp < kMaxAttnSplits; ++sp)
        if (sp < a.splits) s_w[threadIdx.x][sp] = ms[sp] / den;
    }
  }
  __syncthreads();
  // warp w: rows w, w+4, ...; lane: four head dims
  {
    constexpr int RW = kAttnRows / 4;
    float4 acc[RW];
    int grow[RW];   // output row (node * nq + head) of each handled query row, -1 past R
#pragma unroll
    for (int i = 0; i < RW; ++i) {
      acc[i] = make_float4(0.f, 0.f, 0.f, 0.f);
      const int r = rb * kAttnRows + warp + 4 * i;
      grow[i] = r < R ? (r / a.group) * a.nq + g * a.group + r % a.group : -1;
    }
    // splits two at a time: all loads of a pair are issued before any is used
    for (int sp0 = 0; sp0 < a.splits; sp0 += 2) {
      float4 v[2][RW];
#pragma unroll
      for (int q = 0; q < 2; ++q) {
        const float* src = a.o_part + (size_t)(sp0 + q) * rows_total * kAttnD + 4 * lane;
#pragma unroll
        for (int i = 0; i < RW; ++i)
          v[q][i] = (sp0 + q < a.splits && grow[i] >= 0)
                        ? __ldcg(reinterpret_cast<const float4*>(src + (size_t)grow[i] * kAttnD))
                        : make_float4(0.f, 0.f, 0.f, 0.f);
      }
#pragma unroll
      for (int q = 0; q < 2; ++q) {
        if (sp0 + q >= a.splits) break;
#pragma unroll
        for (int i = 0; i < RW; ++i) {
          const float wgt = s_w[warp + 4 * i][sp0 + q];
          acc[i].x += wgt * v[q][i].x;
          acc[i].y += wgt * v[q][i].y;
          acc[i].z += wgt * v[q][i].z;
          acc[i].w += wgt * v[q][i].w;
        }
      }
    }
#pragma unroll
    for (int i = 0; i < RW; ++i)
      if (grow[i] >= 0) store_act4(a.out, (size_t)grow[i] * kAttnD + 4 * lane, a.out_lo_off, acc[i]);
  }
}

// ------------------------------------------------------------ fp32 path
__global__ void __launch_bounds__(128) k_attn_f32(const float* __restrict__ q, const float* __restrict__ kc,
                                                  const float* __restrict__ vc, const unsigned long long* __restrict__ anc,
                                                  int T, int nq, int nkv, int d, int ctx, float scale,
                                                  float* __restrict__ out) {
  __shared__ float qs[128];
  __shared__ float ps[128];
  __shared__ int kpos[128];
  __shared__ float red[32];
  pdl_trigger();
  pdl_wait();
  const int i = blockIdx.x, h = blockIdx.y, g = h / (nq / nkv), tid = threadIdx.x;
  if (tid < d) qs[tid] = q[((size_t)i * nq + h) * d + tid];
  const unsigned long long w0 = anc[2 * i], w1 = anc[2 * i + 1];
  __syncthreads();
  float m = -INFINITY, l = 0.f, acc = 0.f;
  const int n_keys = ctx + T;
  for (int base = 0; base < n_keys; base += blockDim.x) {
    const int kk = base + tid;
    bool valid = kk < n_keys;
    if (valid && kk >= ctx) {
      const int j = kk - ctx;
      valid = ((j < 64 ? (w0 >> j) : (w1 >> (j - 64))) & 1ull) != 0;
    }
    float sc = -INFINITY;
    if (valid) {
      const float* kr = kc + ((size_t)kk * nkv + g) * d;
      float dot = 0.f;
      for (int c = 0; c < d; ++c) dot += qs[c] * kr[c];
      sc = dot * scale;
    }
    const float cmax = block_max(sc, red);
    const float mn = fmaxf(m, cmax);
    const float p = valid ? expf(sc - mn) : 0.f;
    const float corr = (m == -INFINITY) ? 0.f : expf(m - mn);
    const float psum = block_sum(p, red);
    l = l * corr + psum;
    ps[tid] = p;
    kpos[tid] = kk;
    __syncthreads();
    if (tid < d) {
      acc *= corr;
      const int nk = min((int)blockDim.x, n_keys - base);
      for (int k = 0; k < nk; ++k)
        if (ps[k] != 0.f) acc += ps[k] * vc[((size_t)kpos[k] * nkv + g) * d + tid];
    }
    m = mn;
    __syncthreads();
  }
  if (tid < d) out[(size_t)i * nq * d + (size_t)h * d + tid] = acc / l;
}

cudaError_t attn_setup() {
  return cudaFuncSetAttribute(k_attn_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, kAttnSmem);
}

cudaError_t launch_attention(Model& m, const void* kc, const void* vc, int ctx, int T, cudaStream_t st) {
  const auto& c = m.cfg;
  if (c.dtype != OOS_DTYPE_BF16) {
    return launch(m.pdl, k_attn_f32, dim3(T, c.n_q_heads), dim3(128), 0, st, (const float*)m.ws.q, (const float*)kc,
                  (const float*)vc, (const unsigned long long*)m.ws.anc, T, c.n_q_heads, c.n_kv_heads, c.head_dim, ctx,
                  1.0f / sqrtf((float)c.head_dim), (float*)m.ws.attn);
  }
  AttnArgs a;
  a.q = (const __nv_bfloat16*)m.ws.q;
  a.kc = (const __nv_bfloat16*)kc;
  a.vc = (const __nv_bfloat16*)vc;
  a.anc = m.ws.anc;
  a.T = T;
  a.nq = c.n_q_heads;
  a.nkv = c.n_kv_heads;
  a.group = c.n_q_heads / c.n_kv_heads;
  a.ctx = ctx;
  a.cache_blocks = (ctx + kAttnKeys - 1) / kAttnKeys;
  const int R = T * a.group;
  const int RB = (R + kAttnRows - 1) / kAttnRows;
  a.row_blocks = RB;
  // one wave at two blocks per SM (OOS_ATTN_SPLITS overrides, for tuning)
  int splits = (2 * m.num_sms) / (a.nkv * RB);
  if (const char* e = getenv("OOS_ATTN_SPLITS")) splits = atoi(e);
  const int max_splits = a.cache_blocks > 0 ? (a.cache_blocks < kMaxAttnSplits ? a.cache_blocks : kMaxAttnSplits) : 1;
  splits = splits < 1 ? 1 : (splits > max_splits ? max_splits : splits);
  a.splits = splits;
  a.scale_log2 = 1.4426950408889634f / sqrtf((float)kAttnD);
  a.o_part = m.ws.attn_o;
  a.ml_part = m.ws.attn_ml;
  a.cnt = m.ws.attn_cnt;
  a.out = (__nv_bfloat16*)m.ws.attn;
  a.out_lo_off = (size_t)kMaxT * c.n_q_heads * kAttnD;
  return launch(m.pdl, k_attn_tc, dim3(RB, a.nkv, splits), dim3(128), (size_t)kAttnSmem, st, a);
}

}  // namespace oos
