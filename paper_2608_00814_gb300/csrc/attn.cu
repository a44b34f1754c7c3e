// Tree attention of the verify step.
//
// Node i, query head h (kv head g = h / (nq/nkv)) attends to the committed
// cache positions [0, ctx) and to the tree slots ctx + a for every ancestor a
// of i (itself included): softmax(q k / sqrt(d)) v.
//
// bf16 path: split-K over the keys (flash-decoding) inside one thread-block
// cluster.  A block owns 64 query rows of one kv head -- the (node, q-head)
// pairs of the group, so GQA reuses every K/V tile for nq/nkv heads -- and one
// contiguous range of 64-key tiles (cache tiles first, the tree tail last,
// masked with the 128-bit ancestor sets).  The blocks of the different ranges
// of the same rows form one cluster.  K/V tiles are staged in shared memory by
// a 3-deep cp.async ring; scores and P.V run on the tensor cores (mma.sync
// m16n8k16, fp32 accumulate; q as hi + lo bf16 halves) with an online softmax
// in fp32.  Each block then
// leaves its unnormalised O and (max, sum) in its own shared memory, and after
// a cluster barrier every block merges a slice of the rows by log-sum-exp,
// reading the other blocks' shared memory (fixed split order), and writes the
// hi/lo bf16 GEMM input.  The first cache tiles are fetched before the wait on
// the producing kernel: no kernel of the step writes cache positions < ctx.
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
  const __nv_bfloat16* q;   // [T][nq][d] hi halves, lo halves at q_lo_off
  size_t q_lo_off;
  const __nv_bfloat16* kc;  // [cap][nkv][d]
  const __nv_bfloat16* vc;
  const unsigned long long* anc;
  int T, nq, nkv, group, ctx;
  int splits;               // blocks per cluster (key ranges of the same rows)
  int cache_blocks;         // 64-key tiles of the committed cache
  int tiles;                // cache_blocks + tree tiles
  float scale_log2;         // log2(e) / sqrt(d)
  __nv_bfloat16* out;       // [T][nq*d] hi rows, lo rows at out_lo_off
  size_t out_lo_off;
};

// merge staging in the (drained) ring: O rows padded to 136 floats, then (m, l)
constexpr int kAttnOLd = kAttnD + 8;
static_assert(kAttnRows * kAttnOLd * 4 + kAttnRows * 8 <= kAttnSmem, "merge staging exceeds the ring");

OOS_DEV uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
OOS_DEV void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// address of the same shared-memory variable in block `rank` of the cluster
OOS_DEV uint32_t dsmem_addr(const void* p, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_addr(p)), "r"(rank));
  return r;
}
OOS_DEV float4 dsmem_ld4(uint32_t a) {
  float4 v;
  asm volatile("ld.shared::cluster.v4.f32 {%0,%1,%2,%3}, [%4];" : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w) : "r"(a) : "memory");
  return v;
}
OOS_DEV float2 dsmem_ld2(uint32_t a) {
  float2 v;
  asm volatile("ld.shared::cluster.v2.f32 {%0,%1}, [%2];" : "=f"(v.x), "=f"(v.y) : "r"(a) : "memory");
  return v;
}

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
  pdl_trigger();
  const int rb = blockIdx.x, g = blockIdx.y, split = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int R = a.T * a.group;

  // tiles [t0, t1) of this block: cache tiles, then the tree tail
  const int t0 = (int)((long long)split * a.tiles / a.splits);
  const int t1 = (int)((long long)(split + 1) * a.tiles / a.splits);
  const int n_tiles = t1 - t0;
  auto tile_keys = [&](int ti, int& key0, int& key_end, bool& tree) {
    const int t = t0 + ti;
    if (t < a.cache_blocks) {
      key0 = t * kAttnKeys;
      key_end = min(a.ctx, key0 + kAttnKeys);
      tree = false;
    } else {
      key0 = a.ctx + (t - a.cache_blocks) * kAttnKeys;
      key_end = a.ctx + a.T;
      tree = true;
    }
  };
  auto stage_k = [&](int s) { return ring + s * kAttnStageElems; };
  auto stage_v = [&](int s) { return ring + s * kAttnStageElems + kAttnKeys * kAttnLd; };
  auto load = [&](int ti) {
    int k0, ke;
    bool tr;
    tile_keys(ti, k0, ke, tr);
    load_kv_tile(stage_k(ti % kAttnStages), stage_v(ti % kAttnStages), a, g, k0, ke);
  };
  auto issue = [&](int ti) {
    if (ti < n_tiles) load(ti);
    cp_async_commit();
  };

  // Cache tiles do not depend on the producing kernel: fetch the first two
  // before waiting for it.  Tree tiles and Q are read after the wait.
  const bool pre0 = n_tiles > 0 && t0 < a.cache_blocks;
  const bool pre1 = n_tiles > 1 && t0 + 1 < a.cache_blocks;
  if (pre0) load(0);
  if (pre1) load(1);
  pdl_wait();
  if (n_tiles > 0 && !pre0) load(0);
  if (n_tiles > 1 && !pre1) load(1);

  // Q rows (row r -> node r / group, head g*group + r % group), hi halves in the
  // K half and lo halves in the V half of the last ring slot, then kept in
  // registers as mma A fragments: S = q_hi k + q_lo k sees ~16-bit q
  {
    __nv_bfloat16* Qs = stage_k(kAttnStages - 1);
    __nv_bfloat16* Qls = stage_v(kAttnStages - 1);
    for (int c = threadIdx.x; c < kAttnRows * (kAttnD / 8); c += blockDim.x) {
      const int r = c >> 4, col = (c & 15) * 8;
      const int row = rb * kAttnRows + r;
      const bool valid = row < R;
      const int node = valid ? row / a.group : 0, hq = g * a.group + (valid ? row % a.group : 0);
      const __nv_bfloat16* src = a.q + ((size_t)node * a.nq + hq) * kAttnD + col;
      cp_async16(Qs + r * kAttnLd + col, src, valid);
      cp_async16(Qls + r * kAttnLd + col, src + a.q_lo_off, valid);
    }
    cp_async_commit();
    cp_async_wait<0>();   // Q and tiles 0, 1
    __syncthreads();
  }
  uint32_t qf[8][4], qfl[8][4];
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
    const int row = warp * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
    const int col = ks * 16 + (lane >> 4) * 8;
    ldsm_x4(qf[ks], stage_k(kAttnStages - 1) + row * kAttnLd + col);
    ldsm_x4(qfl[ks], stage_v(kAttnStages - 1) + row * kAttnLd + col);
  }
  __syncthreads();
  // tiles 0 and 1 have landed; iteration ti commits one group (tile ti + 2),
  // so wait_group 2 there means tile ti has landed

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
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) mma_bf16(s[nt], qfl[ks], b[nt][0], b[nt][1]);
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) mma_bf16(s[nt], qfl[ks + 1], b[nt][2], b[nt][3]);
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
  __syncthreads();   // every warp is done with the ring

  // quad sums of l, then this block's unnormalised O and (m, l) into its own
  // shared memory
#pragma unroll
  for (int off = 1; off <= 2; off <<= 1) {
    l_lo += __shfl_xor_sync(0xffffffffu, l_lo, off);
    l_hi += __shfl_xor_sync(0xffffffffu, l_hi, off);
  }
  float* so = reinterpret_cast<float*>(smem_raw);     // [64][kAttnOLd]
  float* sml = so + kAttnRows * kAttnOLd;             // [64][2]
  {
    const int lr = warp * 16 + (lane >> 2);
#pragma unroll
    for (int n = 0; n < 16; ++n) {
      const int col = n * 8 + (lane & 3) * 2;
      *reinterpret_cast<float2*>(so + lr * kAttnOLd + col) = make_float2(o[n][0], o[n][1]);
      *reinterpret_cast<float2*>(so + (lr + 8) * kAttnOLd + col) = make_float2(o[n][2], o[n][3]);
    }
    if ((lane & 3) == 0) {
      *reinterpret_cast<float2*>(sml + 2 * lr) = make_float2(m_lo, l_lo);
      *reinterpret_cast<float2*>(sml + 2 * (lr + 8)) = make_float2(m_hi, l_hi);
    }
  }
  cluster_sync();   // every block's partial is in its shared memory

  // block of cluster rank c merges local rows [64c/S, 64(c+1)/S): thread ->
  // (row, four head dims); weights 2^(m_s - M) / sum_s 2^(m_s - M) l_s, summed
  // in split order
  {
    const int S = a.splits;
    const int c = (int)cluster_rank();
    const int lr0 = kAttnRows * c / S, lr1 = kAttnRows * (c + 1) / S;
    for (int idx = threadIdx.x; idx < (lr1 - lr0) * (kAttnD / 4); idx += blockDim.x) {
      const int lr = lr0 + idx / (kAttnD / 4), d4 = (idx % (kAttnD / 4)) * 4;
      const int r = rb * kAttnRows + lr;
      float2 ml[kMaxAttnSplits];
      float M = -INFINITY;
#pragma unroll
      for (int sp = 0; sp < kMaxAttnSplits; ++sp) {
        if (sp < S) {
          ml[sp] = dsmem_ld2(dsmem_addr(sml + 2 * lr, sp));
          M = fmaxf(M, ml[sp].x);
        }
      }
      float4 v[kMaxAttnSplits];
#pragma unroll
      for (int sp = 0; sp < kMaxAttnSplits; ++sp)
        if (sp < S) v[sp] = dsmem_ld4(dsmem_addr(so + lr * kAttnOLd + d4, sp));
      float den = 0.f;
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int sp = 0; sp < kMaxAttnSplits; ++sp) {
        if (sp < S) {
          const float wgt = ml[sp].x == -INFINITY ? 0.f : exp2f(ml[sp].x - M);
          den += wgt * ml[sp].y;
          acc.x += wgt * v[sp].x;
          acc.y += wgt * v[sp].y;
          acc.z += wgt * v[sp].z;
          acc.w += wgt * v[sp].w;
        }
      }
      const float inv = 1.f / den;
      acc.x *= inv;
      acc.y *= inv;
      acc.z *= inv;
      acc.w *= inv;
      if (r < R) {
        const size_t grow = (size_t)(r / a.group) * a.nq + g * a.group + r % a.group;
        store_act4(a.out, grow * kAttnD + d4, a.out_lo_off, acc);
      }
    }
  }
  cluster_sync();   // no block leaves while another may still read its shared memory
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
  a.q_lo_off = (size_t)kMaxT * c.n_q_heads * kAttnD;
  a.kc = (const __nv_bfloat16*)kc;
  a.vc = (const __nv_bfloat16*)vc;
  a.anc = m.ws.anc;
  a.T = T;
  a.nq = c.n_q_heads;
  a.nkv = c.n_kv_heads;
  a.group = c.n_q_heads / c.n_kv_heads;
  a.ctx = ctx;
  a.cache_blocks = (ctx + kAttnKeys - 1) / kAttnKeys;
  a.tiles = a.cache_blocks + (T + kAttnKeys - 1) / kAttnKeys;
  const int R = T * a.group;
  const int RB = (R + kAttnRows - 1) / kAttnRows;
  // one wave at two blocks per SM, at most one cluster of kMaxAttnSplits
  // blocks per row block, no block without a tile
  int splits = (2 * m.num_sms) / (a.nkv * RB);
  splits = splits < 1 ? 1 : (splits > kMaxAttnSplits ? kMaxAttnSplits : splits);
  splits = splits > a.tiles ? a.tiles : splits;
  a.splits = splits;
  a.scale_log2 = 1.4426950408889634f / sqrtf((float)kAttnD);
  a.out = (__nv_bfloat16*)m.ws.attn;
  a.out_lo_off = (size_t)kMaxT * c.n_q_heads * kAttnD;

  cudaLaunchConfig_t lc = {};
  lc.gridDim = dim3(RB, a.nkv, splits);
  lc.blockDim = dim3(128);
  lc.dynamicSmemBytes = (size_t)kAttnSmem;
  lc.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 1;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = splits;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  lc.attrs = attr;
  lc.numAttrs = m.pdl ? 2 : 1;
  return cudaLaunchKernelEx(&lc, k_attn_tc, a);
}

}  // namespace oos
