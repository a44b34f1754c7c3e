// Tree attention of the verify step.
//
// Node i, query head h (kv head g = h / (nq/nkv)) attends to the committed
// cache positions [0, ctx) and to the tree slots ctx + a for every ancestor a
// of i (itself included): softmax(q k / sqrt(d)) v.
//
// bf16 path (tcgen05): split-K over the keys (flash-decoding) inside one
// thread-block cluster.  A block owns 128 query rows of one kv head -- the
// (node, q-head) pairs of the group, so GQA reuses every K/V tile for nq/nkv
// heads, and 128 rows are the MMA's M -- and one contiguous range of 64-key
// tiles (cache tiles first, the tree tail last, masked with the 128-bit
// ancestor sets).  The blocks of the different ranges of the same rows form
// one cluster.  Per tile: S = q K^T on the tensor cores into TMEM (q as hi + lo
// bf16 halves, two MMA passes), a softmax pass with one thread per row reading
// its S row from TMEM, P (bf16) to shared memory, O += P V on the tensor cores
// into TMEM.  The running maximum is moved only when a tile's maximum exceeds
// it by more than 2^8 (O rescaled in TMEM then); otherwise exp2(s - m) stays
// below 256.  V tiles are transposed in shared memory (ldmatrix +
// stmatrix.trans) so that both MMA operands are K-major.  Each block then
// leaves its unnormalised O and (max, sum) in its own shared memory, and after
// a cluster barrier every block merges a slice of the rows by log-sum-exp,
// reading the other blocks' shared memory (fixed split order), and writes the
// hi/lo bf16 GEMM input.  The first cache tiles are fetched before the wait on
// the producing kernel: no kernel of the step writes cache positions < ctx.
//
// fp32 path: one block per (node, head), CUDA cores (small models only).
#include <math.h>
#include <string.h>
#include <stdlib.h>

#include "common.cuh"
#include "internal.h"

namespace oos {

constexpr int kAttnRows = 128;    // query rows per block (tcgen05 M)
constexpr int kAttnKeys = 64;     // keys per tile (S MMA N, P.V MMA K)
constexpr int kAttnD = 128;       // head dim of the bf16 path
// shared memory (bytes): operand tiles in the 128-byte-swizzled K-major layout
constexpr int kQBytes = 2 * kAttnRows * 128;       // 64 of d per 128-byte block: 2 blocks x 128 rows
constexpr int kKBytes = 2 * kAttnKeys * 128;       // K tile: 2 d-blocks x 64 keys
constexpr int kVtBytes = kAttnD * 128;             // V^T tile: 128 d-rows x 64 keys
constexpr int kPBytes = kAttnRows * 128;           // P tile: 128 rows x 64 keys
constexpr int kVrawBytes = 2 * kAttnKeys * 128;   // raw V tile: 2 d-blocks x 64 keys, swizzled
constexpr int kOffQhi = 0;
constexpr int kOffQlo = kOffQhi + kQBytes;
constexpr int kOffK = kOffQlo + kQBytes;           // [2]
constexpr int kOffVt = kOffK + 2 * kKBytes;        // [2]
constexpr int kOffP = kOffVt + 2 * kVtBytes;       // [2]
constexpr int kOffVraw = kOffP + 2 * kPBytes;      // [2]
constexpr int kOffBar = kOffVraw + 2 * kVrawBytes;
constexpr int kAttnSmem = kOffBar + 256 + 1024;    // + barriers + alignment slack
constexpr int kOLd = kAttnD + 4;                   // merge staging row (floats)
constexpr int kOffStage = kOffK;                   // merge staging reuses K, V^T, P
static_assert(kOffStage + kAttnRows * kOLd * 4 + kAttnRows * 8 + kAttnRows * 8 * 4 <= kOffVraw + 2 * kVrawBytes,
              "merge staging");
constexpr int kAttnTmemCols = 256;                 // S[2] (64 columns each), O (128 columns)

struct AttnArgs {
  CUtensorMap qhi, qlo;     // q [node][nq][d] as (d, head in group, kv head, node), hi and lo halves
  CUtensorMap kmap, vmap;   // cache [cap][nkv][d] as (d, kv head, position)
  const unsigned long long* anc;
  int T, nq, nkv, group, ctx;
  int npc;                  // nodes per block: its rows are (node, head in group), npc * group <= 128
  int splits;               // blocks per cluster (key ranges of the same rows)
  int cache_blocks;         // 64-key tiles of the committed cache
  int tiles;                // cache_blocks + tree tiles
  float scale_log2;         // log2(e) / sqrt(d)
  __nv_bfloat16* out;       // [T][nq*d] hi rows, lo rows at out_lo_off
  size_t out_lo_off;
  uint32_t* status;         // step status word (pipeline waits that give up)
  const unsigned char* pf;  // bytes to warm in L2 meanwhile (the next GEMM's weights; may be null)
  size_t pf_bytes;
};

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

OOS_DEV void stsm_x4_t(void* p, const uint32_t (&r)[4]) {
  asm volatile("stmatrix.sync.aligned.m8n8.x4.trans.shared.b16 [%0], {%1,%2,%3,%4};" ::"r"(smem_addr(p)), "r"(r[0]),
               "r"(r[1]), "r"(r[2]), "r"(r[3])
               : "memory");
}
OOS_DEV void cp_async_arrive(uint64_t* bar) {   // arrive once this thread's earlier cp.async have landed
  asm volatile("cp.async.mbarrier.arrive.noinc.shared::cta.b64 [%0];" ::"r"(smem_addr(bar)) : "memory");
}
OOS_DEV void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }
// 2^x by the hardware approximation (relative error ~2^-22; -inf gives +0)
OOS_DEV float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
// 32 lanes x 32 bit, 16 consecutive columns per thread, TMEM <- registers
OOS_DEV void tmem_st16(uint32_t taddr, const float (&v)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(
          taddr),
      "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])), "r"(__float_as_uint(v[3])),
      "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])), "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])),
      "r"(__float_as_uint(v[8])), "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])),
      "r"(__float_as_uint(v[11])), "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])),
      "r"(__float_as_uint(v[14])), "r"(__float_as_uint(v[15]))
      : "memory");
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}
// 16-byte chunk c of row r of a 128-byte-swizzled tile (rows 128 bytes apart,
// 8-row / 1024-byte swizzle atoms, tile base 1024-aligned)
OOS_DEV uint32_t sw128(int r, int c) { return (uint32_t)(r * 128 + ((c ^ (r & 7)) << 4)); }

// sites of the bounded waits (recorded on the status word when one expires)
enum { AW_KEMPTY = 21, AW_VRAW_EMPTY, AW_VFULL, AW_PV_FOR_VT, AW_QFULL, AW_KFULL, AW_SEMPTY, AW_PFULL, AW_VTFULL,
       AW_SFULL, AW_PV_RESCALE, AW_PV_FOR_P, AW_ODONE };
OOS_DEV bool attn_wait(uint64_t* bar, uint32_t parity, volatile int* abort, uint32_t* status, uint32_t site, int ti) {
  if (mbar_wait(bar, parity, abort, status)) return true;
  if (*(volatile uint32_t*)(status + 1) == 0u && (*(volatile uint32_t*)status & ST_TIMEOUT))
    record_timeout(status, site, ti, blockIdx.y, (int)blockIdx.z);
  return false;
}

// Block roles: warp 0 loads (q once, K and raw V per tile, cp.async into the
// swizzled layouts); warp 1 lane 0 issues tcgen05.mma; warps 2..5 run the
// softmax (thread = query row = TMEM lane); warp 6 transposes V tiles.
__global__ void __launch_bounds__(224, 1) k_attn_tc(const __grid_constant__ AttnArgs a) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* sm = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bar = reinterpret_cast<uint64_t*>(sm + kOffBar);
  uint64_t* qfull = bar;            // TMA transaction bytes
  uint64_t* kfull = bar + 1;        // [2] TMA transaction bytes
  uint64_t* kempty = bar + 3;       // [2] S MMAs done
  uint64_t* vfull = bar + 5;        // [2] TMA transaction bytes
  uint64_t* vraw_empty = bar + 7;   // [2] transposer
  uint64_t* vtfull = bar + 9;       // [2] transposer
  uint64_t* sfull = bar + 11;       // [2] S MMAs done
  uint64_t* sempty = bar + 13;      // [2] 4 softmax warps
  uint64_t* pfull = bar + 15;       // [2] 4 softmax warps
  uint64_t* pvdone = bar + 17;      // [2] P.V MMAs done (P and V^T buffers free, O current)
  uint64_t* odone = bar + 19;       // all MMAs done
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bar + 20);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  // the argument block is addressable (its TMA maps are passed by address), so
  // its fields are read once into registers here rather than in the loops
  const int T = a.T, nq = a.nq, group = a.group, ctx = a.ctx, npc = a.npc, n_splits = a.splits;
  const int cache_blocks = a.cache_blocks, n_all = a.tiles;
  const float scale_log2 = a.scale_log2;
  const unsigned long long* anc = a.anc;
  __nv_bfloat16* const out = a.out;
  const size_t out_lo_off = a.out_lo_off;
  uint32_t* status = a.status;
  pdl_trigger();
  const int rb = blockIdx.x, g = blockIdx.y, split = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int rows = npc * group;   // query rows of this block: (node, head in group)

  // tiles [t0, t1) of this block: cache tiles, then the tree tail
  const int t0 = (int)((long long)split * n_all / n_splits);
  const int t1 = (int)((long long)(split + 1) * n_all / n_splits);
  const int n_tiles = t1 - t0;
  auto tile_keys = [&](int ti, int& key0, int& key_end, bool& tree) {
    const int t = t0 + ti;
    if (t < cache_blocks) {
      key0 = t * kAttnKeys;
      key_end = min(ctx, key0 + kAttnKeys);
      tree = false;
    } else {
      key0 = ctx + (t - cache_blocks) * kAttnKeys;
      key_end = ctx + T;
      tree = true;
    }
  };

  if (threadIdx.x == 0) {
    mbar_init(qfull, 1);
    for (int b = 0; b < 2; ++b) {
      mbar_init(&kfull[b], 1);
      mbar_init(&kempty[b], 1);
      mbar_init(&vfull[b], 1);
      mbar_init(&vraw_empty[b], 1);
      mbar_init(&vtfull[b], 1);
      mbar_init(&sfull[b], 1);
      mbar_init(&sempty[b], 4);
      mbar_init(&pfull[b], 4);
      mbar_init(&pvdone[b], 1);
    }
    mbar_init(odone, 1);
    *abort_flag = 0;
    mbar_fence_init();
  }
  if (warp == 2) tmem_alloc(tmem_slot, kAttnTmemCols);
  // q rows past the block's (node, head) rows are MMA padding: zero them (the
  // q loads fill rows [0, rows) only)
  for (int i = threadIdx.x; i < 4 * (kAttnRows - rows) * 8; i += blockDim.x) {
    const int blk = i / ((kAttnRows - rows) * 8), rr = rows + (i / 8) % (kAttnRows - rows), ch = i % 8;
    *reinterpret_cast<uint4*>(sm + kOffQhi + blk * (kAttnRows * 128) + sw128(rr, ch)) = make_uint4(0, 0, 0, 0);
  }
  fence_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t tmem_o = tmem + 2 * kAttnKeys;

  if (warp == 0) {
    // ------------------------------------------------------------ loader (one thread, TMA)
    if (lane == 0) {
      // HBM is nearly idle during attention: pull this block's share of the
      // next GEMM's weights into L2
      if (a.pf) {
        const size_t nb = (size_t)gridDim.x * gridDim.y * gridDim.z;
        const size_t bid = blockIdx.x + (size_t)gridDim.x * (blockIdx.y + (size_t)gridDim.y * blockIdx.z);
        const size_t per = ((a.pf_bytes + nb - 1) / nb + 4095) & ~(size_t)4095;
        const size_t b0 = bid * per;
        const size_t b1 = b0 + per < a.pf_bytes ? b0 + per : a.pf_bytes;
        for (size_t o = b0; o < b1; o += 65536) {
          const uint32_t len = (uint32_t)((b1 - o) < 65536 ? (b1 - o) : 65536);
          asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(a.pf + o), "r"(len & ~15u) : "memory");
        }
      }
      tma_prefetch_desc(&a.kmap);
      tma_prefetch_desc(&a.vmap);
      const uint64_t pol_kv = policy_evict_first();
      auto load_kv = [&](int ti, bool v) {   // K or raw V tile: two 64-wide d blocks of 64 keys
        int k0, ke;
        bool tr;
        tile_keys(ti, k0, ke, tr);
        const int b = ti & 1;
        uint64_t* full = v ? &vfull[b] : &kfull[b];
        unsigned char* dst = sm + (v ? kOffVraw + b * kVrawBytes : kOffK + b * kKBytes);
        mbar_arrive_expect_tx(full, 2 * kAttnKeys * 128);
        tma_load_3d(dst, v ? &a.vmap : &a.kmap, full, 0, g, k0, pol_kv);
        tma_load_3d(dst + kAttnKeys * 128, v ? &a.vmap : &a.kmap, full, 64, g, k0, pol_kv);
      };
      // cache tiles do not depend on the producing kernel: the first two are
      // fetched before waiting for it; tree tiles and q after
      int pre = 0;
      for (int ti = 0; ti < n_tiles && ti < 2; ++ti) {
        int k0, ke;
        bool tr;
        tile_keys(ti, k0, ke, tr);
        if (tr) break;
        load_kv(ti, false);
        load_kv(ti, true);
        pre = ti + 1;
      }
      pdl_wait();
      // q rows of the block's nodes, hi and lo halves, two 64-wide d blocks each
      tma_prefetch_desc(&a.qhi);
      tma_prefetch_desc(&a.qlo);
      const uint64_t pol_q = policy_evict_last();
      mbar_arrive_expect_tx(qfull, 4 * rows * 128);
      const int node0 = rb * npc;
      tma_load_4d(sm + kOffQhi, &a.qhi, qfull, 0, 0, g, node0, pol_q);
      tma_load_4d(sm + kOffQhi + kAttnRows * 128, &a.qhi, qfull, 64, 0, g, node0, pol_q);
      tma_load_4d(sm + kOffQlo, &a.qlo, qfull, 0, 0, g, node0, pol_q);
      tma_load_4d(sm + kOffQlo + kAttnRows * 128, &a.qlo, qfull, 64, 0, g, node0, pol_q);
      for (int ti = pre; ti < n_tiles; ++ti) {
        const int b = ti & 1;
        const uint32_t use = (uint32_t)(ti >> 1);
        if (!attn_wait(&kempty[b], (use & 1u) ^ 1u, abort_flag, status, AW_KEMPTY, ti)) break;
        load_kv(ti, false);
        if (!attn_wait(&vraw_empty[b], (use & 1u) ^ 1u, abort_flag, status, AW_VRAW_EMPTY, ti)) break;
        load_kv(ti, true);
      }
    }
  } else if (warp == 6) {
    // ------------------------------------------------------------ V transposer
    // raw V [key][d] -> V^T [d][key], 128-byte rows of 64 keys, swizzled:
    // ldmatrix reads four 8 x 8 (key x d) blocks, stmatrix.trans writes them as
    // (d x key) rows
    for (int ti = 0; ti < n_tiles; ++ti) {
      const int b = ti & 1;
      const uint32_t use = (uint32_t)(ti >> 1);
      bool ok = true;
      if (lane == 0) {
        ok = attn_wait(&vfull[b], use & 1u, abort_flag, status, AW_VFULL, ti) &&
             attn_wait(&pvdone[b], (use & 1u) ^ 1u, abort_flag, status, AW_PV_FOR_VT, ti);
      }
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) break;
      const unsigned char* vr = sm + kOffVraw + b * kVrawBytes;   // [d block][64 keys][128 B], swizzled
      unsigned char* vt = sm + kOffVt + b * kVtBytes;
      const int i = lane >> 3, j = lane & 7;   // matrix i of the x4, row j of it
#pragma unroll 4
      for (int blk = 0; blk < 32; ++blk) {
        const int kb = blk >> 2;                // 8-key block
        const int db = (blk & 3) * 4 + i;       // 8-d block of matrix i
        uint32_t r[4];
        ldsm_x4(r, vr + (db >> 3) * (kAttnKeys * 128) + sw128(kb * 8 + j, db & 7));
        // row j of the transposed matrix i: d = db*8 + j, keys kb*8 .. kb*8+7
        stsm_x4_t(vt + sw128(db * 8 + j, kb), r);
      }
      fence_async_smem();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&vraw_empty[b]);
        mbar_arrive(&vtfull[b]);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc_s = idesc_bf16_f32(kAttnRows, kAttnKeys);
      constexpr uint32_t idesc_pv = idesc_bf16_f32(kAttnRows, kAttnD);
      bool ok = attn_wait(qfull, 0, abort_flag, status, AW_QFULL, 0);
      fence_async_smem();   // cp.async (generic proxy) writes -> tensor-core reads (async proxy)
      tc_fence_after();
      auto issue_pv = [&](int ti) {
        const int b = ti & 1;
        const uint32_t use = (uint32_t)(ti >> 1);
        if (!attn_wait(&pfull[b], use & 1u, abort_flag, status, AW_PFULL, ti)) return false;
        if (!attn_wait(&vtfull[b], use & 1u, abort_flag, status, AW_VTFULL, ti)) return false;
        fence_async_smem();
        tc_fence_after();
        const uint64_t pd = smem_desc_sw128(smem_addr(sm + kOffP + b * kPBytes));
        const uint64_t vd = smem_desc_sw128(smem_addr(sm + kOffVt + b * kVtBytes));
#pragma unroll
        for (int kk = 0; kk < kAttnKeys / 16; ++kk)
          tc_mma_bf16(tmem_o, pd + 2 * kk, vd + 2 * kk, idesc_pv, (ti > 0 || kk > 0) ? 1u : 0u);
        tc_commit(&pvdone[b]);
        return true;
      };
      for (int ti = 0; ti < n_tiles && ok; ++ti) {
        const int b = ti & 1;
        const uint32_t use = (uint32_t)(ti >> 1);
        if (!attn_wait(&kfull[b], use & 1u, abort_flag, status, AW_KFULL, ti) ||
            !attn_wait(&sempty[b], (use & 1u) ^ 1u, abort_flag, status, AW_SEMPTY, ti)) {
          ok = false;
          break;
        }
        fence_async_smem();
        tc_fence_after();
        const uint32_t ks = smem_addr(sm + kOffK + b * kKBytes);
        const uint32_t d = tmem + b * kAttnKeys;
        // S = q_hi K^T + q_lo K^T over the 128 head dims (two 64-wide blocks)
#pragma unroll
        for (int half = 0; half < 2; ++half) {
          const uint32_t qs = smem_addr(sm + (half ? kOffQlo : kOffQhi));
#pragma unroll
          for (int k = 0; k < kAttnD / 16; ++k) {
            const uint64_t qd = smem_desc_sw128(qs + (k >> 2) * (kAttnRows * 128)) + 2 * (k & 3);
            const uint64_t kd = smem_desc_sw128(ks + (k >> 2) * (kAttnKeys * 128)) + 2 * (k & 3);
            tc_mma_bf16(d, qd, kd, idesc_s, (half > 0 || k > 0) ? 1u : 0u);
          }
        }
        tc_commit(&kempty[b]);
        tc_commit(&sfull[b]);
        if (ti >= 1 && !issue_pv(ti - 1)) ok = false;
      }
      if (ok && n_tiles > 0) issue_pv(n_tiles - 1);
      tc_commit(odone);
    }
  }

  // ------------------------------------------------------------ softmax (warps 2..5)
  float m_used = -INFINITY, l_sum = 0.f;
  const int q4 = warp & 3;
  const int lrow = q4 * 32 + lane;                  // local row = TMEM lane
  const uint32_t lane_off = (uint32_t)(q4 * 32) << 16;
  if (warp >= 2 && warp <= 5) {
    const int node = min(rb * npc + min(lrow, rows - 1) / group, T - 1);
    pdl_wait();
    const unsigned long long anc0 = anc[2 * node], anc1 = anc[2 * node + 1];
    for (int ti = 0; ti < n_tiles; ++ti) {
      const int b = ti & 1;
      const uint32_t use = (uint32_t)(ti >> 1);
      // every wait's outcome is made warp-uniform: the .sync.aligned TMEM
      // accesses and __syncwarp below need the whole warp on one path
      if (!__all_sync(0xffffffffu, attn_wait(&sfull[b], use & 1u, abort_flag, status, AW_SFULL, ti))) break;
      tc_fence_after();
      float s[kAttnKeys];
#pragma unroll
      for (int c = 0; c < kAttnKeys / 16; ++c) {
        float v[16];
        tmem_ld16(tmem + lane_off + b * kAttnKeys + c * 16, v);
#pragma unroll
        for (int i = 0; i < 16; ++i) s[c * 16 + i] = v[i];
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sempty[b]);
      int key0, key_end;
      bool tree;
      tile_keys(ti, key0, key_end, tree);
      // masked keys: past the cache end of a partial tile, tree slots that are
      // not ancestors of this node (a tile-uniform branch: full cache tiles skip it)
      if (tree || key_end < key0 + kAttnKeys) {
        // key key0 + i is valid when i < n_valid and, for tree tile tt, bit i of
        // the node's ancestor word tt (tree slot 64 tt + i) is set
        const int n_valid = key_end - key0;
        const unsigned long long word = !tree ? ~0ull : ((key0 - ctx) < 64 ? anc0 : anc1);
#pragma unroll
        for (int i = 0; i < kAttnKeys; ++i)
          if (i >= n_valid || !((word >> i) & 1ull)) s[i] = -INFINITY;
      }
      // row maximum of the raw scores, four independent chains
      float mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
      for (int i = 0; i < kAttnKeys; i += 4) {
        mx[0] = fmaxf(mx[0], s[i]);
        mx[1] = fmaxf(mx[1], s[i + 1]);
        mx[2] = fmaxf(mx[2], s[i + 2]);
        mx[3] = fmaxf(mx[3], s[i + 3]);
      }
      const float tmax = fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])) * scale_log2;   // scale > 0
      // move the running maximum only when this tile exceeds it by 2^8
      // (a lane that moves its maximum rescales its O row; the whole warp takes
      // part in the TMEM accesses, lanes that keep theirs scale by 1)
      const bool move = tmax > m_used + 8.f;
      const bool rescale = move && m_used != -INFINITY;
      if (__any_sync(0xffffffffu, rescale)) {
        // O holds P.V of tiles < ti: wait for the last of them, then rescale
        {
          const int pb = (ti - 1) & 1;
          if (!__all_sync(0xffffffffu, attn_wait(&pvdone[pb], (uint32_t)((ti - 1) >> 1) & 1u, abort_flag, status,
                                                 AW_PV_RESCALE, ti)))
            break;
          tc_fence_after();
          const float f = rescale ? exp2f(m_used - tmax) : 1.f;
#pragma unroll 1
          for (int c = 0; c < kAttnD / 16; ++c) {
            float v[16];
            tmem_ld16(tmem_o + lane_off + c * 16, v);
#pragma unroll
            for (int i = 0; i < 16; ++i) v[i] *= f;
            tmem_st16(tmem_o + lane_off + c * 16, v);
          }
          l_sum *= f;
          tc_fence_before();
        }
      }
      if (move) m_used = tmax;
      // p = 2^(s * scale - m): one FMA and one ex2 per score; a masked score
      // (-inf) gives 0; a row with nothing unmasked yet (m = -inf) gives 0
      uint32_t pk[kAttnKeys / 2];
      float ps[4] = {0.f, 0.f, 0.f, 0.f};
      const bool live = m_used != -INFINITY;
      const float neg_m = live ? -m_used : 0.f;
#pragma unroll
      for (int i = 0; i < kAttnKeys; i += 2) {
        const float p0 = live ? ex2_approx(fmaf(s[i], scale_log2, neg_m)) : 0.f;
        const float p1 = live ? ex2_approx(fmaf(s[i + 1], scale_log2, neg_m)) : 0.f;
        const __nv_bfloat162 pp = __floats2bfloat162_rn(p0, p1);
        // the sum uses the rounded weights that P.V multiplies
        ps[(i >> 1) & 3] += __low2float(pp) + __high2float(pp);
        pk[i / 2] = *reinterpret_cast<const uint32_t*>(&pp);
      }
      const float psum = (ps[0] + ps[1]) + (ps[2] + ps[3]);
      l_sum += psum;
      // P buffer b is free once P.V of tile ti - 2 has completed
      if (!__all_sync(0xffffffffu, attn_wait(&pvdone[b], (use & 1u) ^ 1u, abort_flag, status, AW_PV_FOR_P, ti))) break;
      unsigned char* prow = sm + kOffP + b * kPBytes;
#pragma unroll
      for (int c = 0; c < 8; ++c)
        *reinterpret_cast<uint4*>(prow + sw128(lrow, c)) = make_uint4(pk[4 * c], pk[4 * c + 1], pk[4 * c + 2], pk[4 * c + 3]);
      fence_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&pfull[b]);
    }
  }

  // every role is done with the rings once all MMAs have completed
  if (warp >= 2 && warp <= 5) attn_wait(odone, 0, abort_flag, status, AW_ODONE, n_tiles);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  // this block's unnormalised O rows and (m, l) into its own shared memory
  float* so = reinterpret_cast<float*>(sm + kOffStage);   // [128][kOLd]
  float* sml = so + kAttnRows * kOLd;                     // [128][2]
  if (warp >= 2 && warp <= 5) {
#pragma unroll 1
    for (int c = 0; c < kAttnD / 16; ++c) {
      float v[16];
      tmem_ld16(tmem_o + lane_off + c * 16, v);
#pragma unroll
      for (int i = 0; i < 16; i += 4)
        *reinterpret_cast<float4*>(so + lrow * kOLd + c * 16 + i) = make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
    }
    *reinterpret_cast<float2*>(sml + 2 * lrow) = make_float2(*abort_flag ? -INFINITY : m_used, l_sum);
  }
  tc_fence_before();
  cluster_sync();   // every block's partial is in its shared memory

  // block of cluster rank c merges local rows [rows c/S, rows (c+1)/S): first
  // each row's split weights 2^(m_s - M) / sum_s 2^(m_s - M) l_s, then thread ->
  // (row, four head dims) sums the splits' O in split order
  {
    const int S = n_splits;
    const int c = (int)cluster_rank();
    const int lr0 = rows * c / S, lr1 = rows * (c + 1) / S;
    float* sw = sml + 2 * kAttnRows;   // [row - lr0][kMaxAttnSplits], this block only
    if (threadIdx.x < lr1 - lr0) {
      const int lr = lr0 + threadIdx.x;
      float2 ml[kMaxAttnSplits];
      float M = -INFINITY;
#pragma unroll
      for (int sp = 0; sp < kMaxAttnSplits; ++sp) {
        if (sp < S) {
          ml[sp] = dsmem_ld2(dsmem_addr(sml + 2 * lr, sp));
          M = fmaxf(M, ml[sp].x);
        }
      }
      float den = 0.f;
#pragma unroll
      for (int sp = 0; sp < kMaxAttnSplits; ++sp) {
        if (sp < S) {
          ml[sp].x = ml[sp].x == -INFINITY ? 0.f : exp2f(ml[sp].x - M);
          den += ml[sp].x * ml[sp].y;
        }
      }
      const float inv = den > 0.f ? 1.f / den : 0.f;
#pragma unroll
      for (int sp = 0; sp < kMaxAttnSplits; ++sp)
        if (sp < S) sw[threadIdx.x * kMaxAttnSplits + sp] = ml[sp].x * inv;
    }
    __syncthreads();
    for (int idx = threadIdx.x; idx < (lr1 - lr0) * (kAttnD / 4); idx += blockDim.x) {
      const int lr = lr0 + idx / (kAttnD / 4), d4 = (idx % (kAttnD / 4)) * 4;
      const int node = rb * npc + lr / group;
      float4 v[kMaxAttnSplits];
#pragma unroll
      for (int sp = 0; sp < kMaxAttnSplits; ++sp)
        if (sp < S) v[sp] = dsmem_ld4(dsmem_addr(so + lr * kOLd + d4, sp));
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int sp = 0; sp < kMaxAttnSplits; ++sp) {
        if (sp < S) {
          const float wgt = sw[(lr - lr0) * kMaxAttnSplits + sp];
          acc.x += wgt * v[sp].x;
          acc.y += wgt * v[sp].y;
          acc.z += wgt * v[sp].z;
          acc.w += wgt * v[sp].w;
        }
      }
      if (node < T) {
        const size_t grow = (size_t)node * nq + g * group + lr % group;
        store_act4(out, grow * kAttnD + d4, out_lo_off, acc);
      }
    }
  }
  cluster_sync();   // no block leaves while another may still read its shared memory
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, kAttnTmemCols);
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

int attn_nodes_per_block(int group) { return group >= kAttnRows ? 1 : kAttnRows / group; }

bool attn_encode_q_maps(Model& m) {
  const auto& c = m.cfg;
  const int group = c.n_q_heads / c.n_kv_heads;
  // q [node][nq][d] viewed as (d, head in group, kv head, node); a box is the
  // (node, head in group) rows of one kv head, 64 of d at a time
  const uint64_t dims[4] = {(uint64_t)kAttnD, (uint64_t)group, (uint64_t)c.n_kv_heads, (uint64_t)kMaxT};
  const uint64_t strides[3] = {(uint64_t)kAttnD * 2, (uint64_t)group * kAttnD * 2, (uint64_t)c.n_q_heads * kAttnD * 2};
  const uint32_t box[4] = {64, (uint32_t)group, 1, (uint32_t)attn_nodes_per_block(group)};
  const __nv_bfloat16* q = (const __nv_bfloat16*)m.ws.q;
  return encode_bf16_map(&m.qmap_hi, q, 4, dims, strides, box) &&
         encode_bf16_map(&m.qmap_lo, q + (size_t)kMaxT * c.n_q_heads * kAttnD, 4, dims, strides, box);
}

// clusters of `sp` attention blocks resident at once on this device (occupancy query, cached)
static int attn_max_clusters(int sp) {
  static int cached[kMaxAttnSplits + 1] = {0};
  if (sp < 1 || sp > kMaxAttnSplits) return 0;
  if (cached[sp] == 0) {
    cudaLaunchConfig_t lc = {};
    lc.gridDim = dim3(1, 1, sp);
    lc.blockDim = dim3(224);
    lc.dynamicSmemBytes = (size_t)kAttnSmem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 1;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = sp;
    lc.attrs = attr;
    lc.numAttrs = 1;
    int n = 0;
    cached[sp] = cudaOccupancyMaxActiveClusters(&n, (const void*)k_attn_tc, &lc) == cudaSuccess && n > 0 ? n : -1;
  }
  return cached[sp];
}

cudaError_t attn_setup() {
  return cudaFuncSetAttribute(k_attn_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, kAttnSmem);
}

cudaError_t launch_attention(Model& m, int layer, const void* kc, const void* vc, int ctx, int T, cudaStream_t st) {
  const auto& c = m.cfg;
  if (c.dtype != OOS_DTYPE_BF16) {
    return launch(m.pdl, k_attn_f32, dim3(T, c.n_q_heads), dim3(128), 0, st, (const float*)m.ws.q, (const float*)kc,
                  (const float*)vc, (const unsigned long long*)m.ws.anc, T, c.n_q_heads, c.n_kv_heads, c.head_dim, ctx,
                  1.0f / sqrtf((float)c.head_dim), (float*)m.ws.attn);
  }
  AttnArgs a;
  memset(&a, 0, sizeof(a));
  a.qhi = m.qmap_hi;
  a.qlo = m.qmap_lo;
  // this call's cache, (d, kv head, position) over the ctx + T valid positions:
  // a tile reaching past them reads zeros (and masks them)
  {
    if ((int)m.kv_maps.size() != c.n_layers) m.kv_maps.assign(c.n_layers, Model::KvMaps());
    Model::KvMaps& km = m.kv_maps[layer];
    if (km.k != kc || km.v != vc || km.extent != ctx + T) {
      const uint64_t dims[3] = {(uint64_t)kAttnD, (uint64_t)c.n_kv_heads, (uint64_t)(ctx + T)};
      const uint64_t strides[2] = {(uint64_t)kAttnD * 2, (uint64_t)c.n_kv_heads * kAttnD * 2};
      const uint32_t box[3] = {64, 1, (uint32_t)kAttnKeys};
      if (!encode_bf16_map(&km.kmap, kc, 3, dims, strides, box) ||
          !encode_bf16_map(&km.vmap, vc, 3, dims, strides, box)) {
        km.k = km.v = nullptr;
        return cudaErrorInvalidValue;
      }
      km.k = kc;
      km.v = vc;
      km.extent = ctx + T;
    }
    a.kmap = km.kmap;
    a.vmap = km.vmap;
  }
  a.anc = m.ws.anc;
  a.T = T;
  a.nq = c.n_q_heads;
  a.nkv = c.n_kv_heads;
  a.group = c.n_q_heads / c.n_kv_heads;
  a.npc = attn_nodes_per_block(a.group);
  a.ctx = ctx;
  a.cache_blocks = (ctx + kAttnKeys - 1) / kAttnKeys;
  a.tiles = a.cache_blocks + (T + kAttnKeys - 1) / kAttnKeys;
  const int RB = (T + a.npc - 1) / a.npc;
  // The most splits (one cluster of them per row block and kv head) such that
  // every cluster is resident at once -- one wave -- and no block is without a tile.
  const int pairs = a.nkv * RB;
  int splits = 1;
  for (int sp = kMaxAttnSplits; sp >= 1; --sp) {
    if (sp > a.tiles || pairs * sp > m.num_sms) continue;
    if (attn_max_clusters(sp) >= pairs) {
      splits = sp;
      break;
    }
  }
  a.splits = splits;
  a.scale_log2 = 1.4426950408889634f / sqrtf((float)kAttnD);
  a.out = (__nv_bfloat16*)m.ws.attn;
  a.out_lo_off = (size_t)kMaxT * c.n_q_heads * kAttnD;
  a.status = m.ws.status;
  // the O-projection weights of this layer, [H][nq*d] bf16, contiguous
  a.pf = (const unsigned char*)m.layers[layer].w_o;
  a.pf_bytes = (size_t)c.hidden * c.n_q_heads * kAttnD * 2;

  cudaLaunchConfig_t lc = {};
  lc.gridDim = dim3(RB, a.nkv, splits);
  lc.blockDim = dim3(224);
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
