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
// bf16 halves, two MMA passes, with q itself held in TMEM as the A operand), a
// softmax pass with one thread per row reading its S row from TMEM and writing
// P (bf16) back into TMEM, O += P V on the tensor cores into TMEM (P the A
// operand from TMEM).  Two threads issue the MMAs, one the S products and one
// the P.V products, so neither waits behind the other's barriers.  The
// running maximum is moved only when a tile's maximum exceeds
// it by more than 2^8 (O rescaled in TMEM then); otherwise exp2(s - m) stays
// below 256.  V tiles enter the P.V MMA as they arrive ([key][d], d
// contiguous: the MN-major operand layout), through a ring of kKvStages K and V
// tiles that keeps several tile loads in flight.  Each block then
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
constexpr int kVBytes = 2 * kAttnKeys * 128;       // V tile: 2 d-blocks x 64 keys
constexpr int kKvStages = 4;                       // K and V tiles in flight
constexpr int kOffQhi = 0;
constexpr int kOffQlo = kOffQhi + kQBytes;
constexpr int kOffK = kOffQlo + kQBytes;           // [kKvStages]
constexpr int kOffV = kOffK + kKvStages * kKBytes; // [kKvStages]
constexpr int kOffBar = kOffV + kKvStages * kVBytes;
constexpr int kAttnSmem = kOffBar + 256 + 1024;    // + barriers + alignment slack
constexpr int kAttnThreads = 224;                  // 7 warps, roles below
constexpr int kOLd = kAttnD + 4;                   // merge staging row (floats)
constexpr int kOffStage = kOffK;                   // merge staging reuses K and V
static_assert(kOffStage + kAttnRows * kOLd * 4 + kAttnRows * 8 + kAttnRows * 8 * 4 <= kOffBar, "merge staging");
static_assert(kAttnSmem <= 227 * 1024, "shared memory per block");
// TMEM columns (lane = query row): S[2] fp32 scores of a tile, O fp32, q hi
// and lo as packed bf16 pairs along d, P[2] as packed bf16 pairs along the keys
constexpr int kTmS = 0;                            // [2] x 64
constexpr int kTmO = 2 * kAttnKeys;                // 128
constexpr int kTmQ = kTmO + kAttnD;                // [hi, lo] x 64
constexpr int kTmP = kTmQ + 2 * (kAttnD / 2);      // [2] x 32
constexpr int kAttnTmemCols = 512;                 // power of two >= kTmP + 64
static_assert(kTmP + 2 * (kAttnKeys / 2) <= kAttnTmemCols, "TMEM columns");

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

// D[tmem] (+)= A[tmem] * B[smem]: A (M = 128 rows, one per lane) as packed
// bf16 pairs, K index 2c and 2c + 1 in column c (low half first)
OOS_DEV void tc_mma_bf16_ts(uint32_t tmem_d, uint32_t tmem_a, uint64_t bdesc, uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(tmem_d),
      "r"(tmem_a), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Shared-memory descriptor of an MN-major operand in the 128-byte-swizzled
// layout: 64 consecutive MN elements (bf16) per 128-byte row, one row per K
// index, 8-row / 1024-byte swizzle atoms.  `lbo` is the byte distance between
// consecutive 64-element MN blocks, the stride between 8-row K groups is 1024.
OOS_DEV uint64_t smem_desc_sw128_mn(uint32_t saddr, uint32_t lbo) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)(1024u >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
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
// 32 lanes x 32 bit, 16 consecutive columns per thread, TMEM <- raw words
OOS_DEV void tmem_st16u(uint32_t taddr, const uint32_t* v) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(
          taddr),
      "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]), "r"(v[9]),
      "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15])
      : "memory");
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}
// 16-byte chunk c of row r of a 128-byte-swizzled tile (rows 128 bytes apart,
// 8-row / 1024-byte swizzle atoms, tile base 1024-aligned)
OOS_DEV uint32_t sw128(int r, int c) { return (uint32_t)(r * 128 + ((c ^ (r & 7)) << 4)); }

// sites of the bounded waits (recorded on the status word when one expires)
enum { AW_KEMPTY = 21, AW_VEMPTY, AW_QFULL, AW_KFULL, AW_SEMPTY, AW_PFULL, AW_VFULL, AW_SFULL, AW_PV_RESCALE,
       AW_PV_FOR_P, AW_ODONE };
OOS_DEV bool attn_wait(uint64_t* bar, uint32_t parity, volatile int* abort, uint32_t* status, uint32_t site, int ti) {
  if (mbar_wait(bar, parity, abort, status)) return true;
  if (*(volatile uint32_t*)(status + 1) == 0u && (*(volatile uint32_t*)status & ST_TIMEOUT))
    record_timeout(status, site, ti, blockIdx.y, (int)blockIdx.z);
  return false;
}

// Block roles: warp 0 lane 0 loads (q once, K and V per tile, by TMA into the
// swizzled layouts); warp 1 lane 0 issues the S MMAs, warp 6 lane 0 the P.V
// MMAs; warps 2..5 run the softmax (thread = query row = TMEM lane).
__global__ void __launch_bounds__(kAttnThreads, 1) k_attn_tc(const __grid_constant__ AttnArgs a) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* sm = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bar = reinterpret_cast<uint64_t*>(sm + kOffBar);
  uint64_t* qfull = bar;                      // TMA transaction bytes
  uint64_t* kfull = bar + 1;                  // [kKvStages] TMA transaction bytes
  uint64_t* kempty = kfull + kKvStages;       // [kKvStages] S MMAs done
  uint64_t* vfull = kempty + kKvStages;       // [kKvStages] TMA transaction bytes
  uint64_t* vempty = vfull + kKvStages;       // [kKvStages] P.V MMAs done
  uint64_t* sfull = vempty + kKvStages;       // [2] S MMAs done
  uint64_t* sempty = sfull + 2;               // [2] 4 softmax warps
  uint64_t* pfull = sempty + 2;               // [2] 4 softmax warps
  uint64_t* pvdone = pfull + 2;               // [2] P.V MMAs done (P buffer free, O current)
  uint64_t* odone = pvdone + 2;               // all MMAs of both issuers done
  uint64_t* qtm = odone + 1;                  // 4 softmax warps: q rows are in TMEM
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(qtm + 1);
  static_assert((1 + 4 * kKvStages + 10) * 8 + 8 <= 256, "barrier block");
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
    for (int s = 0; s < kKvStages; ++s) {
      mbar_init(&kfull[s], 1);
      mbar_init(&kempty[s], 1);
      mbar_init(&vfull[s], 1);
      mbar_init(&vempty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&sfull[b], 1);
      mbar_init(&sempty[b], 4);
      mbar_init(&pfull[b], 4);
      mbar_init(&pvdone[b], 1);
    }
    mbar_init(odone, 2);   // both MMA issuers
    mbar_init(qtm, 4);
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
  const uint32_t tmem_o = tmem + kTmO;

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
      auto load_kv = [&](int ti, bool v) {   // K or V tile: two 64-wide d blocks of 64 keys
        int k0, ke;
        bool tr;
        tile_keys(ti, k0, ke, tr);
        const int s = ti % kKvStages;
        uint64_t* full = v ? &vfull[s] : &kfull[s];
        unsigned char* dst = sm + (v ? kOffV + s * kVBytes : kOffK + s * kKBytes);
        mbar_arrive_expect_tx(full, 2 * kAttnKeys * 128);
        tma_load_3d(dst, v ? &a.vmap : &a.kmap, full, 0, g, k0, pol_kv);
        tma_load_3d(dst + kAttnKeys * 128, v ? &a.vmap : &a.kmap, full, 64, g, k0, pol_kv);
      };
      // cache tiles do not depend on the producing kernel: the first stages
      // are fetched before waiting for it; tree tiles and q after
      int pre = 0;
      for (int ti = 0; ti < n_tiles && ti < kKvStages; ++ti) {
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
        const int st = ti % kKvStages;
        const uint32_t use = (uint32_t)(ti / kKvStages);
        if (!attn_wait(&kempty[st], (use & 1u) ^ 1u, abort_flag, status, AW_KEMPTY, ti)) break;
        load_kv(ti, false);
        if (!attn_wait(&vempty[st], (use & 1u) ^ 1u, abort_flag, status, AW_VEMPTY, ti)) break;
        load_kv(ti, true);
      }
    }
  } else if (warp == 1 || warp == 6) {
    // ------------------------------------------------------------ MMA issuers
    // warp 1 lane 0 issues S = q K^T, warp 6 lane 0 issues O += P V: two
    // threads, so that neither kind waits behind the other's barriers and the
    // tensor cores always have queued work.  Operands reach the tensor cores
    // through the async proxy only: q, K and V by TMA, P from threads that
    // fence before they arrive on pfull (the zeroed q padding rows were fenced
    // before the block barrier).  Descriptors: the start address is the low
    // field (16-byte units), so a byte offset o inside an operand region is
    // added as o >> 4.
    if (lane == 0 && warp == 1) {
      constexpr uint32_t idesc_s = idesc_bf16_f32(kAttnRows, kAttnKeys);
      bool ok = attn_wait(qtm, 0, abort_flag, status, AW_QFULL, 0);
      tc_fence_after();
      const uint64_t kdesc0 = smem_desc_sw128(smem_addr(sm + kOffK));
      // S buffer ti & 1 is free once the softmax has read tile ti - 2's scores,
      // before P of tile ti - 2 is ready: the scores run ahead of the softmax
      for (int ti = 0; ti < n_tiles && ok; ++ti) {
        const int b = ti & 1;
        const uint32_t use = (uint32_t)(ti >> 1);
        const int st = ti % kKvStages;
        if (!attn_wait(&kfull[st], (uint32_t)(ti / kKvStages) & 1u, abort_flag, status, AW_KFULL, ti) ||
            !attn_wait(&sempty[b], (use & 1u) ^ 1u, abort_flag, status, AW_SEMPTY, ti))
          break;
        tc_fence_after();
        const uint64_t kd0 = kdesc0 + (uint64_t)((st * kKBytes) >> 4);
        const uint32_t d = tmem + kTmS + b * kAttnKeys;
        // S = q_hi K^T + q_lo K^T over the 128 head dims: q from TMEM (8
        // columns = 16 of d per MMA), K from the two 64-wide d blocks (32 bytes
        // of d per MMA)
#pragma unroll
        for (int half = 0; half < 2; ++half) {
#pragma unroll
          for (int k = 0; k < kAttnD / 16; ++k) {
            const uint64_t kd = kd0 + (uint64_t)(((k >> 2) * (kAttnKeys * 128)) >> 4) + 2 * (k & 3);
            tc_mma_bf16_ts(d, tmem + kTmQ + half * (kAttnD / 2) + 8 * k, kd, idesc_s, (half > 0 || k > 0) ? 1u : 0u);
          }
        }
        tc_commit(&kempty[st]);
        tc_commit(&sfull[b]);
      }
      tc_commit(odone);
    } else if (lane == 0 && warp == 6) {
      constexpr uint32_t idesc_pv = idesc_bf16_f32(kAttnRows, kAttnD) | (1u << 16);   // B (V) MN-major
      // V tile: d blocks of 64 (8 KB apart) along N, 16 keys (2 KB) per MMA along K
      const uint64_t vdesc0 = smem_desc_sw128_mn(smem_addr(sm + kOffV), kAttnKeys * 128);
      for (int ti = 0; ti < n_tiles; ++ti) {
        const int b = ti & 1;
        const uint32_t use = (uint32_t)(ti >> 1);
        const int st = ti % kKvStages;
        if (!attn_wait(&pfull[b], use & 1u, abort_flag, status, AW_PFULL, ti) ||
            !attn_wait(&vfull[st], (uint32_t)(ti / kKvStages) & 1u, abort_flag, status, AW_VFULL, ti))
          break;
        tc_fence_after();
        const uint32_t pt = tmem + kTmP + b * (kAttnKeys / 2);   // P: 8 columns = 16 keys per MMA
        const uint64_t vd = vdesc0 + (uint64_t)((st * kVBytes) >> 4);
#pragma unroll
        for (int kk = 0; kk < kAttnKeys / 16; ++kk)
          tc_mma_bf16_ts(tmem_o, pt + 8 * kk, vd + (uint64_t)((kk * 16 * 128) >> 4), idesc_pv, (ti > 0 || kk > 0) ? 1u : 0u);
        tc_commit(&pvdone[b]);
        tc_commit(&vempty[st]);
      }
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
    // this thread's q row (hi, lo) from the TMA tile into TMEM, the S MMAs'
    // A operand: 16 columns per store = 32 of d as bf16 pairs; padding rows
    // past the block's rows are the zeroed shared-memory rows
    const bool qok = __all_sync(0xffffffffu, attn_wait(qfull, 0, abort_flag, status, AW_QFULL, 0));
    if (qok) {
#pragma unroll
      for (int part = 0; part < 8; ++part) {   // (hi/lo, 64-wide d block, half of its 8 chunks)
        const unsigned char* qb = sm + ((part >> 2) ? kOffQlo : kOffQhi) + ((part >> 1) & 1) * (kAttnRows * 128);
        uint32_t w[16];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          const uint4 v = *reinterpret_cast<const uint4*>(qb + sw128(lrow, (part & 1) * 4 + c));
          w[4 * c] = v.x;
          w[4 * c + 1] = v.y;
          w[4 * c + 2] = v.z;
          w[4 * c + 3] = v.w;
        }
        tmem_st16u(tmem + lane_off + kTmQ + part * 16, w);
      }
    }
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive(qtm);
    for (int ti = 0; ti < (qok ? n_tiles : 0); ++ti) {
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
        tmem_ld16(tmem + lane_off + kTmS + b * kAttnKeys + c * 16, v);
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
      // P into TMEM, the P.V MMAs' A operand (key pairs, 32 columns)
      tmem_st16u(tmem + lane_off + kTmP + b * (kAttnKeys / 2), pk);
      tmem_st16u(tmem + lane_off + kTmP + b * (kAttnKeys / 2) + 16, pk + 16);
      tc_fence_before();
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
    lc.blockDim = dim3(kAttnThreads);
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
  lc.blockDim = dim3(kAttnThreads);
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
