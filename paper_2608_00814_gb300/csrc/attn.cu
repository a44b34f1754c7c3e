// Tree attention of the verify step.
//
// Node i, query head h (kv head g = h / (nq/nkv)) attends to the committed
// cache positions [0, ctx) and to the tree slots ctx + a for every ancestor a
// of i (itself included): softmax(q k / sqrt(d)) v.  The tree's own K/V sit in
// slots ctx .. ctx+T-1 right after the committed ones, so the keys of one
// (node, head) are a masked prefix of the contiguous slot range [0, ctx+T).
//
// bf16 path (tcgen05), split-K over the keys inside one thread-block cluster.
// A block owns up to 128 query rows of one kv head -- the (node, q-head) pairs
// of the group, so GQA reuses every K/V tile for nq/nkv heads, and 128 rows
// are the MMA's M -- and one contiguous range of 128-key tiles of [0, ctx+T).
// The blocks of the different ranges of the same rows form one cluster (up to
// 16 blocks, non-portable size, chosen so that every cluster is resident at
// once).  Per tile:
//   - S = q K^T on the tensor cores into TMEM, N = 128 keys, q as hi + lo
//     bf16 halves (two MMA chains), the A operand straight from the shared
//     memory TMA staged it in;
//   - softmax, one thread per query row: the row's S from TMEM, the valid-key
//     mask (cache keys, then the node's ancestors), exp2, and P (bf16 pairs)
//     written back over the first 64 columns of the same S buffer;
//   - O += P V on the tensor cores (P the A operand from TMEM, V in the
//     MN-major layout TMA writes, [key][d]).
// Two threads issue the MMAs (S, and P.V) so neither waits behind the other's
// barriers; K/V tiles come by TMA through a two-stage ring.  The running
// maximum moves only when a tile exceeds it by more than 2^8 (O is rescaled
// in TMEM then).
// Merge: each block stages its unnormalised O rows and (max, sum) in its own
// shared memory, and one thread copies each owner's rows into that owner's
// shared memory (bulk copies that complete on the owner's barrier, no round
// trips); the owner adds the splits by log-sum-exp in split order
// (deterministic) and writes the hi/lo bf16 GEMM input.
//
// The slot range is read through tensor maps over the cache's whole capacity,
// and ctx comes from device memory (written by the step's tree preparation), so
// one launch serves any ctx.  Keys past ctx + T in the last tile are masked,
// and their V rows are zeroed in shared memory before the P.V product, so
// whatever the cache holds there cannot reach the output.
//
// fp32 path: one block per (node, head), CUDA cores (small models only).
#include <math.h>
#include <string.h>
#include <stdlib.h>

#include "common.cuh"
#include "internal.h"

// Step timeline (built only with -DOOS_TIMELINE, see timeline.py): per block
// of the last attention launch, the globaltimer at entry (0), at the end of the
// loader's dependency wait (1), when q has landed (2), at the start and end of
// the softmax of tiles 0..5 (3 + 2t, 4 + 2t), when all MMAs are done (15), when
// the merge rows are staged (21), past the cluster barrier (22), when this
// block's rows have been copied out (16) and its own rows received (17), and at
// exit (18); slots 19 and 20 hold the block's tile count and the split count.
#ifdef OOS_TIMELINE
namespace oos {
__device__ unsigned long long g_tl_attn[2048][24];
}
#define TL_ATTN(ev)                                                                      \
  do {                                                                                   \
    const unsigned bid_ = blockIdx.x + gridDim.x * (blockIdx.y + gridDim.y * blockIdx.z); \
    if (bid_ < 2048) oos::g_tl_attn[bid_][ev] = oos::globaltimer();                      \
  } while (0)
#define TL_ATTN_VAL(ev, v)                                                               \
  do {                                                                                   \
    const unsigned bid_ = blockIdx.x + gridDim.x * (blockIdx.y + gridDim.y * blockIdx.z); \
    if (bid_ < 2048) oos::g_tl_attn[bid_][ev] = (unsigned long long)(v);                 \
  } while (0)
#else
#define TL_ATTN(ev) \
  do {              \
  } while (0)
#define TL_ATTN_VAL(ev, v) \
  do {                     \
  } while (0)
#endif

namespace oos {

constexpr int kAttnRows = 128;     // query rows per block (tcgen05 M)
constexpr int kAttnKeys = 128;     // keys per tile (N of the S MMAs)
constexpr int kAttnD = 128;        // head dim of the bf16 path
constexpr int kKvStages = 2;       // K and V tiles in flight
// shared memory (bytes): operand tiles in the 128-byte-swizzled layout TMA
// writes: per tile two 64-wide d blocks of 128 keys x 128 bytes
constexpr int kDBlock = kAttnKeys * 128;                  // 16 KB
constexpr int kTileBytes = 2 * kDBlock;                   // 32 KB
constexpr int kOffK = 0;                                  // [kKvStages]
constexpr int kOffV = kOffK + kKvStages * kTileBytes;     // [kKvStages]
constexpr int kMaxSplits = 16;
constexpr int kRecvRows = kAttnRows + kMaxSplits;         // >= splits * ceil(rows / splits)
// a merge row: the unnormalised O row (128 fp32), then (max, sum), padded to 16 bytes
constexpr int kMergeLd = kAttnD + 4;                      // floats
constexpr int kMergeRowBytes = kMergeLd * 4;              // 528
constexpr int kOffStage = kOffK;                          // merge: this block's rows, staged over the K/V ring
constexpr int kOffRecv = kOffV + kKvStages * kTileBytes;  // merge: rows copied in by the splits [slot][kMergeLd]
constexpr int kOffWgt = kOffRecv + kRecvRows * kMergeRowBytes;   // merge weights [owned row][split]
constexpr int kOffBar = kOffWgt + kAttnRows * kMaxSplits * 4;
static_assert(kAttnRows * kMergeRowBytes <= kKvStages * 2 * kTileBytes, "merge staging");
static_assert(4 * kAttnRows * 128 <= kRecvRows * kMergeRowBytes, "q staging in the receive buffer");
static_assert((kOffRecv & 1023) == 0, "swizzled q staging is 1024-aligned");
constexpr int kAttnSmem = kOffBar + 256 + 1024;           // + barriers + alignment slack
constexpr int kAttnThreads = 224;                         // 7 warps, roles below
static_assert(kAttnSmem <= 227 * 1024, "shared memory per block");
static_assert(kMaxSplits <= 16, "cluster size");
// TMEM columns (lane = query row): S[2] fp32 scores of a tile (P, bf16 pairs,
// overwrites the first 64 columns of its S buffer), O fp32
constexpr int kTmS = 0;                            // [2] x 128
constexpr int kTmO = 2 * kAttnKeys;                // 128
constexpr int kAttnTmemCols = 512;                 // allocation unit: a power of two
static_assert(kTmO + kAttnD <= kAttnTmemCols, "TMEM columns");

struct AttnArgs {
  CUtensorMap kmap, vmap;   // cache [capacity][nkv][d] as (d, kv head, slot)
  CUtensorMap qhi, qlo;     // q [node][nq][d] as (d, head in group, kv head, node), hi and lo halves
  const unsigned long long* anc;
  const int* ctx_dev;       // committed positions of the step (written by tree preparation)
  int T, nq, group;
  int npc;                  // nodes per block: its rows are (node, head in group), npc * group <= 128
  int splits;               // blocks per cluster (key ranges of the same rows)
  float scale_log2;         // log2(e) / sqrt(d)
  __nv_bfloat16* out;       // [T][nq*d] hi rows, lo rows at out_lo_off
  size_t out_lo_off;
  uint32_t* status;         // step status word (pipeline waits that give up)
};

OOS_DEV uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// not .aligned: the threads of a warp may arrive at different points
OOS_DEV void cluster_arrive_release() { asm volatile("barrier.cluster.arrive.release;" ::: "memory"); }
OOS_DEV void cluster_wait_acquire() { asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory"); }
// address of the same shared-memory location in block `rank` of the cluster
OOS_DEV uint32_t dsmem_addr(const void* p, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_addr(p)), "r"(rank));
  return r;
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
// 16-byte chunk c of row r of a 128-byte-swizzled tile (rows 128 bytes apart,
// 8-row / 1024-byte swizzle atoms, tile base 1024-aligned)
OOS_DEV uint32_t sw128(int r, int c) { return (uint32_t)(r * 128 + ((c ^ (r & 7)) << 4)); }
// 32 lanes x 32 bit, 16 consecutive columns per thread, TMEM <- raw words
OOS_DEV void tmem_st16u(uint32_t taddr, const uint32_t* v) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(
          taddr),
      "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]), "r"(v[9]),
      "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15])
      : "memory");
}
OOS_DEV void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
// 32 lanes x 32 bit, 32 consecutive columns per thread, without waiting: the
// caller issues several, then tmem_wait_ld_regs over every register loaded
OOS_DEV void tmem_ld32_nowait(uint32_t taddr, float* v) {
  uint32_t* r = reinterpret_cast<uint32_t*>(v);
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}
// wait for the thread's outstanding TMEM loads; the empty statements after it
// make every later use of v[0..n) depend on the wait
template <int N>
OOS_DEV void tmem_wait_ld_regs(float (&v)[N]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < N; ++i) asm volatile("" : "+f"(v[i]));
}
// all 128 columns of one lane row starting at taddr
OOS_DEV void tmem_ld128(uint32_t taddr, float (&v)[128]) {
#pragma unroll
  for (int c = 0; c < 4; ++c) tmem_ld32_nowait(taddr + c * 32, v + c * 32);
  tmem_wait_ld_regs(v);
}
// bulk copy shared::cta -> shared::cluster of another block, completing bytes on
// that block's mbarrier (both remote addresses from mapa)
OOS_DEV void bulk_copy_to_peer(uint32_t dst, const void* src, uint32_t bytes, uint32_t remote_bar) {
  asm volatile("cp.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   dst),
               "r"(smem_addr(src)), "r"(bytes), "r"(remote_bar)
               : "memory");
}
OOS_DEV void bulk_commit_and_wait_read() {
  asm volatile("cp.async.bulk.commit_group;\n\tcp.async.bulk.wait_group.read 0;" ::: "memory");
}

// 128-bit masks as (lo: bits 0..63, hi: bits 64..127)
OOS_DEV void shr128(unsigned long long lo, unsigned long long hi, int s, unsigned long long& rlo,
                    unsigned long long& rhi) {
  if (s >= 128) { rlo = 0; rhi = 0; }
  else if (s >= 64) { rlo = s == 64 ? hi : hi >> (s - 64); rhi = 0; }
  else if (s == 0) { rlo = lo; rhi = hi; }
  else { rlo = (lo >> s) | (hi << (64 - s)); rhi = hi >> s; }
}
OOS_DEV void shl128(unsigned long long lo, unsigned long long hi, int s, unsigned long long& rlo,
                    unsigned long long& rhi) {
  if (s >= 128) { rlo = 0; rhi = 0; }
  else if (s >= 64) { rhi = s == 64 ? lo : lo << (s - 64); rlo = 0; }
  else if (s == 0) { rlo = lo; rhi = hi; }
  else { rhi = (hi << s) | (lo >> (64 - s)); rlo = lo << s; }
}

// sites of the bounded waits (recorded on the status word when one expires)
enum { AW_KEMPTY = 21, AW_VEMPTY, AW_QFULL, AW_KFULL, AW_SFREE, AW_PFULL, AW_VFULL, AW_SFULL, AW_PV_RESCALE,
       AW_VZERO };
OOS_DEV bool attn_wait(uint64_t* bar, uint32_t parity, volatile int* abort, uint32_t* status, uint32_t site, int ti) {
  if (mbar_wait(bar, parity, abort, status)) return true;
  if (*(volatile uint32_t*)(status + 1) == 0u && (*(volatile uint32_t*)status & ST_TIMEOUT))
    record_timeout(status, site, ti, blockIdx.y, (int)blockIdx.z);
  return false;
}
// a CTA's own copies or MMAs draining after an abort: bounded by the default limit
OOS_DEV void drain_wait(uint64_t* bar, uint32_t parity) {
  const unsigned long long t0 = globaltimer();
  while (!mbar_test(smem_addr(bar), parity) && globaltimer() - t0 < kWaitLimitNs) {
  }
}

// Block roles: warp 0 lane 0 loads K and V tiles (TMA into the swizzled
// layouts); warp 1 lane 0 issues the S MMAs, warp 6 lane 0 the P.V MMAs;
// warps 2..5 run the softmax (thread = query row = TMEM lane); all warps take
// part in the merge.
// F16: the KV cache (and q) are IEEE binary16 -- every product runs in f16;
// otherwise bf16.
template <bool F16>
__global__ void __launch_bounds__(kAttnThreads, 1) k_attn_tc(const __grid_constant__ AttnArgs a) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* sm = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bar = reinterpret_cast<uint64_t*>(sm + kOffBar);
  uint64_t* kfull = bar;          // [2] TMA transaction bytes
  uint64_t* kempty = bar + 2;     // [2] S MMAs of the stage's tile done
  uint64_t* vfull = bar + 4;      // [2] TMA transaction bytes
  uint64_t* vempty = bar + 6;     // [2] P.V MMAs of the stage's tile done
  uint64_t* sfull = bar + 8;      // [2] S MMAs done
  uint64_t* pfull = bar + 10;     // [2] 4 softmax warps: P written
  uint64_t* pvdone = bar + 12;    // [2] P.V MMAs done (S/P buffer free, O current)
  uint64_t* odone = bar + 15;     // both MMA issuers done
  uint64_t* recv_full = bar + 16; // merge: every split's rows for this block copied in (transaction bytes)
  uint64_t* qfull = bar + 17;     // q tile landed (transaction bytes)
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bar + 18);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  static_assert(18 * 8 + 8 <= 256, "barrier block");

  if (threadIdx.x == 0) TL_ATTN(0);
  const int T = a.T, nq = a.nq, G = a.group, npc = a.npc, S = a.splits;
  const float scale_log2 = a.scale_log2;
  uint32_t* status = a.status;
  const int rb = blockIdx.x, g = blockIdx.y, split = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int node0 = rb * npc;
  const int rows = npc * G;                                   // query rows of the block
  const int vrows = max(0, min(rows, (T - node0) * G));       // rows of real nodes

  // Committed positions of the step.  The step's tree preparation wrote them
  // and has completed: every kernel of the step lets its dependents launch
  // only after its own dependency wait, so when this kernel starts the kernel
  // two launches back and everything before it are complete.
  const int ctx = *a.ctx_dev;
  const int n_all = (ctx + T + kAttnKeys - 1) / kAttnKeys;   // tiles over slots [0, ctx + T)
  const int t0 = (int)((long long)split * n_all / S);
  const int n_tiles = (int)((long long)(split + 1) * n_all / S) - t0;
  // merge: rows [0, vrows) are dealt to the S blocks of the cluster, block j
  // owning rows [vrows j / S, vrows (j+1) / S)
  const int n_max = (vrows + S - 1) / S;
  const int lr0_mine = (int)((long long)vrows * split / S);
  const int n_mine = (int)((long long)vrows * (split + 1) / S) - lr0_mine;

  if (threadIdx.x == 0) {
    for (int s = 0; s < 2; ++s) {
      mbar_init(&kfull[s], 1);
      mbar_init(&kempty[s], 1);
      mbar_init(&vfull[s], 1);
      mbar_init(&vempty[s], 1);
      mbar_init(&sfull[s], 1);
      mbar_init(&pfull[s], 4);
      mbar_init(&pvdone[s], 1);
    }
    mbar_init(odone, 2);
    mbar_init(recv_full, 1);
    mbar_init(qfull, 1);
    // every split copies its rows of this block in: S * n_mine merge rows
    mbar_arrive_expect_tx(recv_full, (uint32_t)(S * n_mine * kMergeRowBytes));
    *abort_flag = 0;
    mbar_fence_init();
  }
  if (warp == 2) tmem_alloc(tmem_slot, kAttnTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  // Another block may copy into this block's receive buffer only once the
  // block runs, its receive barrier is armed and the S MMAs no longer read the
  // q tile staged in that buffer: every thread arrives on the cluster barrier
  // when it is past that point (the softmax threads after the last tile's S,
  // the others now), and every block waits for the whole cluster before its
  // merge copies.
  if (warp < 2 || warp > 5) cluster_arrive_release();
  const uint32_t tmem = *tmem_slot;
  const uint32_t tmem_o = tmem + kTmO;

  if (warp == 0) {
    // ------------------------------------------------------------ loader (one thread, TMA)
    if (lane == 0) {
      tma_prefetch_desc(&a.kmap);
      tma_prefetch_desc(&a.vmap);
      const uint64_t pol_kv = policy_evict_first();
      auto load = [&](int ti, bool v) {   // K or V tile: two 64-wide d blocks of 128 slots
        const int st = ti & 1;
        const int key0 = (t0 + ti) * kAttnKeys;
        uint64_t* full = v ? &vfull[st] : &kfull[st];
        unsigned char* dst = sm + (v ? kOffV : kOffK) + st * kTileBytes;
        mbar_arrive_expect_tx(full, kTileBytes);
        tma_load_3d(dst, v ? &a.vmap : &a.kmap, full, 0, g, key0, pol_kv);
        tma_load_3d(dst + kDBlock, v ? &a.vmap : &a.kmap, full, 64, g, key0, pol_kv);
      };
      // tiles of committed slots only do not depend on the producing kernel:
      // the first stages are fetched before waiting for it
      int nk = 0, nv = 0;   // K and V tiles issued
      while (nk < n_tiles && nk < kKvStages && (t0 + nk + 1) * kAttnKeys <= ctx) {
        load(nk, false);
        load(nk, true);
        ++nk;
        ++nv;
      }
      pdl_wait();
      pdl_trigger();
      TL_ATTN(1);
      // q rows of the block's nodes, hi and lo halves, two 64-wide d blocks
      // each, staged in the (still unused) receive buffer
      tma_prefetch_desc(&a.qhi);
      tma_prefetch_desc(&a.qlo);
      {
        const uint64_t pol_q = policy_evict_last();
        unsigned char* qs = sm + kOffRecv;
        mbar_arrive_expect_tx(qfull, (uint32_t)(4 * rows * 128));
        tma_load_4d(qs, &a.qhi, qfull, 0, 0, g, node0, pol_q);
        tma_load_4d(qs + kAttnRows * 128, &a.qhi, qfull, 64, 0, g, node0, pol_q);
        tma_load_4d(qs + 2 * kAttnRows * 128, &a.qlo, qfull, 0, 0, g, node0, pol_q);
        tma_load_4d(qs + 3 * kAttnRows * 128, &a.qlo, qfull, 64, 0, g, node0, pol_q);
      }
      for (int ti = nk; ti < n_tiles; ++ti) {
        const int st = ti & 1;
        const uint32_t use = (uint32_t)(ti >> 1);
        if (!attn_wait(&kempty[st], (use & 1u) ^ 1u, abort_flag, status, AW_KEMPTY, ti)) break;
        load(ti, false);
        ++nk;
        if (!attn_wait(&vempty[st], (use & 1u) ^ 1u, abort_flag, status, AW_VEMPTY, ti)) break;
        load(ti, true);
        ++nv;
      }
      // every copy this thread issued has landed before the block can exit,
      // whoever gave up (immediate on the normal path, where all were consumed)
      for (int ti = nk > 2 ? nk - 2 : 0; ti < nk; ++ti) drain_wait(&kfull[ti & 1], (uint32_t)(ti >> 1) & 1u);
      for (int ti = nv > 2 ? nv - 2 : 0; ti < nv; ++ti) drain_wait(&vfull[ti & 1], (uint32_t)(ti >> 1) & 1u);
      drain_wait(qfull, 0);
    }
  } else if (warp == 1 || warp == 6) {
    // ------------------------------------------------------------ MMA issuers
    // Operands reach the tensor cores through the async proxy only: q, K and
    // V by TMA, P from threads that wait for their TMEM stores before they
    // arrive, the zeroed V rows fenced by the threads that wrote them.
    // Descriptors: the start address is the low field (16-byte units), so a
    // byte offset o inside an operand region is added as o >> 4.
    if (lane == 0 && warp == 1) {
      constexpr uint32_t idesc_s = F16 ? idesc_f16_f32(kAttnRows, kAttnKeys) : idesc_bf16_f32(kAttnRows, kAttnKeys);
      bool ok = attn_wait(qfull, 0, abort_flag, status, AW_QFULL, 0);
      TL_ATTN(2);
      tc_fence_after();
      const uint64_t kdesc0 = smem_desc_sw128(smem_addr(sm + kOffK));
      // q as staged by TMA: [hi d0, hi d1, lo d0, lo d1], each 128 rows x 128
      // bytes in the swizzled K-major layout (rows of padding nodes hold
      // whatever the q buffer holds; every row of S, P and O is its own)
      const uint64_t qdesc0 = smem_desc_sw128(smem_addr(sm + kOffRecv));
      for (int ti = 0; ti < n_tiles && ok; ++ti) {
        const int b = ti & 1;
        const uint32_t use = (uint32_t)(ti >> 1);
        // S buffer b holds P of tile ti - 2 until that tile's P.V is done
        if (!attn_wait(&kfull[b], use & 1u, abort_flag, status, AW_KFULL, ti) ||
            !attn_wait(&pvdone[b], (use & 1u) ^ 1u, abort_flag, status, AW_SFREE, ti))
          break;
        tc_fence_after();
        const uint64_t kd0 = kdesc0 + (uint64_t)((b * kTileBytes) >> 4);
        const uint32_t d = tmem + kTmS + b * kAttnKeys;
        // S = q_hi K^T + q_lo K^T over the 128 head dims: q and K both from
        // their two 64-wide d blocks (32 bytes of d per MMA)
#pragma unroll
        for (int half = 0; half < 2; ++half) {
#pragma unroll
          for (int k = 0; k < kAttnD / 16; ++k) {
            const uint64_t kd = kd0 + (uint64_t)(((k >> 2) * kDBlock) >> 4) + 2 * (k & 3);
            const uint64_t qd = qdesc0 + (uint64_t)(((2 * half + (k >> 2)) * (kAttnRows * 128)) >> 4) + 2 * (k & 3);
            tc_mma_bf16(d, qd, kd, idesc_s, (half > 0 || k > 0) ? 1u : 0u);
          }
        }
        tc_commit(&kempty[b]);
        tc_commit(&sfull[b]);
      }
      tc_commit(odone);
    } else if (lane == 0 && warp == 6) {
      constexpr uint32_t idesc_pv =
          (F16 ? idesc_f16_f32(kAttnRows, kAttnD) : idesc_bf16_f32(kAttnRows, kAttnD)) | (1u << 16);   // B (V) MN-major
      // V tile: d blocks of 64 (kDBlock apart) along N, 16 keys (2 KB) per MMA along K
      const uint64_t vdesc0 = smem_desc_sw128_mn(smem_addr(sm + kOffV), kDBlock);
      for (int ti = 0; ti < n_tiles; ++ti) {
        const int b = ti & 1;
        const uint32_t use = (uint32_t)(ti >> 1);
        if (!attn_wait(&pfull[b], use & 1u, abort_flag, status, AW_PFULL, ti) ||
            !attn_wait(&vfull[b], use & 1u, abort_flag, status, AW_VFULL, ti))
          break;
        tc_fence_after();
        const uint32_t pt = tmem + kTmS + b * kAttnKeys;   // P: 8 columns = 16 keys per MMA
        const uint64_t vd = vdesc0 + (uint64_t)((b * kTileBytes) >> 4);
#pragma unroll
        for (int kk = 0; kk < kAttnKeys / 16; ++kk)
          tc_mma_bf16_ts(tmem_o, pt + 8 * kk, vd + (uint64_t)((kk * 16 * 128) >> 4), idesc_pv,
                         (ti > 0 || kk > 0) ? 1u : 0u);
        tc_commit(&pvdone[b]);
        tc_commit(&vempty[b]);
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
    const bool real = lrow < vrows;
    const int node = real ? node0 + lrow / G : node0;
    unsigned long long anc0 = 0ull, anc1 = 0ull;
    bool waited = false;
    // Iteration -1 is a dry pass of the tile body, run before the dependency
    // wait while the block has nothing else to do: it brings the body's code
    // into the SM's instruction caches (the step's other kernels have evicted
    // it since the previous layer), reads whatever S buffer 0 holds, and
    // discards everything -- no wait, store, arrive or state update.
#pragma unroll 1
    for (int ti = -1; ti < n_tiles; ++ti) {
      asm volatile("" : "+r"(ti));   // one loop body for every iteration: none is specialised
      const bool dry = ti < 0;         // warp-uniform
      if (ti == 0) {
        pdl_wait();
        pdl_trigger();
        waited = true;
        anc0 = a.anc[2 * node];
        anc1 = a.anc[2 * node + 1];
      }
      const int tt = dry ? 0 : ti;
      const int b = tt & 1;
      const uint32_t use = (uint32_t)(tt >> 1);
      if (!dry) {
        // every wait's outcome is made warp-uniform: the .sync.aligned TMEM
        // accesses and __syncwarp below need the whole warp on one path
        if (!__all_sync(0xffffffffu, attn_wait(&sfull[b], use & 1u, abort_flag, status, AW_SFULL, ti))) break;
        tc_fence_after();
      }
      const int key0 = dry ? ctx : (t0 + ti) * kAttnKeys;
      if (!dry && warp == 2 && lane == 0 && ti < 6) TL_ATTN(3 + 2 * ti);
      // valid keys of this row in the tile: committed slots, then the tree
      // slots of the node's ancestors (slot ctx + j for ancestor j); slots at
      // or past ctx + T are never ancestors (the dry pass takes the masked path)
      const bool full_tile = !dry && key0 + kAttnKeys <= ctx;   // tile-uniform
      unsigned long long mlo = ~0ull, mhi = ~0ull;
      if (!full_tile) {
        const int c = max(0, ctx - key0);                 // leading committed slots (< 128)
        unsigned long long tlo, thi;
        if (key0 >= ctx) shr128(anc0, anc1, key0 - ctx, tlo, thi);
        else shl128(anc0, anc1, c, tlo, thi);
        const unsigned long long clo = c >= 64 ? ~0ull : (c == 0 ? 0ull : (~0ull >> (64 - c)));
        const unsigned long long chi = c <= 64 ? 0ull : (~0ull >> (128 - c));
        mlo = clo | tlo;
        mhi = chi | thi;
      }
      // the row's 128 scores, masked keys at -inf
      float sv[kAttnKeys];
      tmem_ld128(tmem + lane_off + kTmS + b * kAttnKeys, sv);
      if (!full_tile) {
#pragma unroll
        for (int i = 0; i < kAttnKeys; ++i)
          if (!((((i < 64) ? mlo : mhi) >> (i & 63)) & 1ull)) sv[i] = -INFINITY;
      }
      float mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
      for (int i = 0; i < kAttnKeys; ++i) mx[i & 3] = fmaxf(mx[i & 3], sv[i]);
      const float tmax = fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])) * scale_log2;   // scale > 0
      // move the running maximum only when this tile exceeds it by 2^8 (a
      // lane that moves its maximum rescales its O row; the whole warp takes
      // part in the TMEM accesses, lanes that keep theirs scale by 1)
      const bool move = !dry && tmax > m_used + 8.f;
      const bool rescale = move && m_used != -INFINITY;
      if (__any_sync(0xffffffffu, rescale)) {
        // O holds P.V of tiles < ti: wait for the last of them, then rescale
        const int pb = (ti - 1) & 1;
        if (!__all_sync(0xffffffffu, attn_wait(&pvdone[pb], (uint32_t)((ti - 1) >> 1) & 1u, abort_flag, status,
                                               AW_PV_RESCALE, ti)))
          break;
        tc_fence_after();
        const float f = rescale ? exp2f(m_used - tmax) : 1.f;
#pragma unroll 1
        for (int c = 0; c < kAttnD / 32; ++c) {   // 32 columns at a time: the scores stay in registers
          float ov[32];
          tmem_ld32_nowait(tmem_o + lane_off + c * 32, ov);
          tmem_wait_ld_regs(ov);
#pragma unroll
          for (int i = 0; i < 32; ++i) ov[i] *= f;
          tmem_st16u(tmem_o + lane_off + c * 32, reinterpret_cast<const uint32_t*>(ov));
          tmem_st16u(tmem_o + lane_off + c * 32 + 16, reinterpret_cast<const uint32_t*>(ov + 16));
          tmem_wait_st();
        }
        l_sum *= f;
      }
      if (move) m_used = tmax;
      // p = 2^(s * scale - m): one FMA and one ex2 per score; a masked score
      // (-inf) gives 0, and a row with nothing valid yet (m = -inf) gives 0
      uint32_t pk[kAttnKeys / 2];
      float ps[4] = {0.f, 0.f, 0.f, 0.f};
      const bool live = dry || m_used != -INFINITY;
      const float neg_m = (live && !dry) ? -m_used : 0.f;
#pragma unroll
      for (int i = 0; i < kAttnKeys; i += 2) {
        const float p0 = live ? ex2_approx(fmaf(sv[i], scale_log2, neg_m)) : 0.f;
        const float p1 = live ? ex2_approx(fmaf(sv[i + 1], scale_log2, neg_m)) : 0.f;
        // P in the operand format of V; the sum uses the rounded weights that P.V multiplies
        if constexpr (F16) {
          const __half2 pp = __floats2half2_rn(p0, p1);
          ps[(i >> 1) & 3] += __low2float(pp) + __high2float(pp);
          pk[i / 2] = *reinterpret_cast<const uint32_t*>(&pp);
        } else {
          const __nv_bfloat162 pp = __floats2bfloat162_rn(p0, p1);
          ps[(i >> 1) & 3] += __low2float(pp) + __high2float(pp);
          pk[i / 2] = *reinterpret_cast<const uint32_t*>(&pp);
        }
      }
      if (dry) {   // the weights count as used, so that the dry pass computes them
#pragma unroll
        for (int i = 0; i < kAttnKeys / 2; ++i) asm volatile("" ::"r"(pk[i]));
        asm volatile("" ::"f"(ps[0]), "f"(ps[1]), "f"(ps[2]), "f"(ps[3]));
        continue;
      }
      l_sum += (ps[0] + ps[1]) + (ps[2] + ps[3]);
      // slots at or past ctx + T in this tile hold whatever the cache holds
      // there: zero their V rows (P is 0 for them, but 0 * NaN is not 0)
      const int n_ok = ctx + T - key0;                   // tile-uniform
      if (n_ok < kAttnKeys) {
        if (!__all_sync(0xffffffffu, attn_wait(&vfull[b], use & 1u, abort_flag, status, AW_VZERO, ti))) break;
        if (lrow >= n_ok) {
          unsigned char* vt = sm + kOffV + b * kTileBytes + lrow * 128;
#pragma unroll
          for (int c = 0; c < 8; ++c) {
            *reinterpret_cast<uint4*>(vt + c * 16) = make_uint4(0, 0, 0, 0);
            *reinterpret_cast<uint4*>(vt + kDBlock + c * 16) = make_uint4(0, 0, 0, 0);
          }
          fence_async_smem();
        }
      }
      // P over the first 64 columns of S buffer b (S of this tile is read)
#pragma unroll
      for (int part = 0; part < 4; ++part) tmem_st16u(tmem + lane_off + kTmS + b * kAttnKeys + part * 16, pk + part * 16);
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&pfull[b]);
      if (warp == 2 && lane == 0 && ti < 6) TL_ATTN(4 + 2 * ti);
    }
    if (!waited) {   // no tile: the dependency wait is still owed
      pdl_wait();
      pdl_trigger();
    }
    // the S MMAs are done with the staged q (every S this thread waited for);
    // after an abort an S MMA may still read it while a peer's merge rows
    // arrive -- the step has failed then, and only values are affected
    cluster_arrive_release();
    // every role is done with the rings and TMEM once all MMAs have completed;
    // both issuers always commit this barrier, and TMEM must not be released
    // under a running MMA, so the wait is not cut short by the handle's limit
    drain_wait(odone, 0);
    if (warp == 2 && lane == 0) TL_ATTN(15);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();

  // ------------------------------------------------------------ merge
  // Each block stages its O row, max and sum of every real row in its own
  // shared memory (over the K/V ring, idle now), and one thread copies each
  // owner's rows into slots split * n_max .. of that owner's receive buffer
  // (bulk copies, completing on the owner's receive barrier).  The owner then
  // adds the S splits of its rows by log-sum-exp, in split order.
  float* stage = reinterpret_cast<float*>(sm + kOffStage);   // [row][kMergeLd]
  const float* recv = reinterpret_cast<const float*>(sm + kOffRecv);
  float* wgt = reinterpret_cast<float*>(sm + kOffWgt);
  const bool have_o = n_tiles > 0 && !*abort_flag;   // block-uniform after the barrier
  if (warp >= 2 && warp <= 5) {
    float ov[kAttnD];
    if (have_o) {
      tmem_ld128(tmem_o + lane_off, ov);
    } else {
#pragma unroll
      for (int i = 0; i < kAttnD; ++i) ov[i] = 0.f;
    }
    if (lrow < vrows) {
      float* row = stage + (size_t)lrow * kMergeLd;
#pragma unroll
      for (int i = 0; i < kAttnD; i += 4) *reinterpret_cast<float4*>(row + i) = make_float4(ov[i], ov[i + 1], ov[i + 2], ov[i + 3]);
      *reinterpret_cast<float4*>(row + kAttnD) = make_float4(have_o ? m_used : -INFINITY, have_o ? l_sum : 0.f, 0.f, 0.f);
      fence_async_smem();   // the rows are read by the bulk-copy engine
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) TL_ATTN(21);
  cluster_wait_acquire();   // every block of the cluster runs and has armed its receive barrier
  if (threadIdx.x == 0) TL_ATTN(22);
  if (threadIdx.x == 0) {
    for (int j = 0; j < S; ++j) {
      const int r0 = (int)((long long)vrows * j / S), r1 = (int)((long long)vrows * (j + 1) / S);
      if (r1 > r0)
        bulk_copy_to_peer(dsmem_addr(sm + kOffRecv + (size_t)split * n_max * kMergeRowBytes, (uint32_t)j),
                          stage + (size_t)r0 * kMergeLd, (uint32_t)((r1 - r0) * kMergeRowBytes),
                          dsmem_addr(recv_full, (uint32_t)j));
    }
    bulk_commit_and_wait_read();   // the staged rows have been read before this block moves on
  }
  if (threadIdx.x == 0) TL_ATTN(16);
  // this block's rows from every split.  Every block copies its rows even
  // after an abort, so this wait ends; it is not cut short by the handle's
  // limit, because the block must not exit while copies into it are in flight.
  drain_wait(recv_full, 0);
  if (threadIdx.x == 0) TL_ATTN(17);
  {
    // split weights of every owned row: 2^(m_s - M) / sum_s 2^(m_s - M) l_s
    // (every split's value of a row is loaded before any is used: the loops
    // run over the largest split count, guarded, so they unroll)
    if (threadIdx.x < n_mine) {
      const int i = threadIdx.x;
      float ms[kMaxSplits], ls[kMaxSplits];
      float M = -INFINITY;
#pragma unroll
      for (int s2 = 0; s2 < kMaxSplits; ++s2) {
        if (s2 < S) {
          const float2 ml = *reinterpret_cast<const float2*>(recv + (size_t)(s2 * n_max + i) * kMergeLd + kAttnD);
          ms[s2] = ml.x;
          ls[s2] = ml.y;
          M = fmaxf(M, ml.x);
        }
      }
      float den = 0.f, w[kMaxSplits];
#pragma unroll
      for (int s2 = 0; s2 < kMaxSplits; ++s2) {
        if (s2 < S) {
          w[s2] = ms[s2] == -INFINITY ? 0.f : exp2f(ms[s2] - M);
          den += w[s2] * ls[s2];
        }
      }
      const float inv = den > 0.f ? 1.f / den : 0.f;
#pragma unroll
      for (int s2 = 0; s2 < kMaxSplits; ++s2)
        if (s2 < S) wgt[i * kMaxSplits + s2] = w[s2] * inv;
    }
    __syncthreads();
    for (int idx = threadIdx.x; idx < n_mine * (kAttnD / 4); idx += blockDim.x) {
      const int i = idx / (kAttnD / 4), d4 = (idx % (kAttnD / 4)) * 4;
      float4 v[kMaxSplits];
#pragma unroll
      for (int s2 = 0; s2 < kMaxSplits; ++s2)
        if (s2 < S) v[s2] = *reinterpret_cast<const float4*>(recv + (size_t)(s2 * n_max + i) * kMergeLd + d4);
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int s2 = 0; s2 < kMaxSplits; ++s2) {
        if (s2 < S) {
          const float ws = wgt[i * kMaxSplits + s2];
          acc.x += ws * v[s2].x;
          acc.y += ws * v[s2].y;
          acc.z += ws * v[s2].z;
          acc.w += ws * v[s2].w;
        }
      }
      const int lr = lr0_mine + i;
      const size_t grow = (size_t)(node0 + lr / G) * nq + g * G + lr % G;
      store_act4(a.out, grow * kAttnD + d4, a.out_lo_off, acc);
    }
  }
  if (threadIdx.x == 0) {
    TL_ATTN(18);
    TL_ATTN_VAL(19, n_tiles);
    TL_ATTN_VAL(20, S);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, kAttnTmemCols);
  }
}

// ------------------------------------------------------------ fp32 path
__global__ void __launch_bounds__(128) k_attn_f32(const float* __restrict__ q, const float* __restrict__ kc,
                                                  const float* __restrict__ vc, const unsigned long long* __restrict__ anc,
                                                  int T, int nq, int nkv, int d, const int32_t* __restrict__ ctx_dev,
                                                  float scale, float* __restrict__ out) {
  __shared__ float qs[128];
  __shared__ float ps[128];
  __shared__ int kpos[128];
  __shared__ float red[32];
  pdl_wait();
  pdl_trigger();
  const int ctx = *ctx_dev;
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
  const bool f16 = c.kv_f16 != 0;
  return encode_bf16_map(&m.qmap_hi, q, 4, dims, strides, box, f16) &&
         encode_bf16_map(&m.qmap_lo, q + (size_t)kMaxT * c.n_q_heads * kAttnD, 4, dims, strides, box, f16);
}

// clusters of `sp` attention blocks resident at once on this device (occupancy query, cached)
static int attn_max_clusters(int sp) {
  static int cached[kMaxSplits + 1] = {0};
  if (sp < 1 || sp > kMaxSplits) return 0;
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
    cached[sp] = cudaOccupancyMaxActiveClusters(&n, (const void*)k_attn_tc<false>, &lc) == cudaSuccess && n > 0 ? n : -1;
    cudaGetLastError();
  }
  return cached[sp];
}

template <bool F16>
static cudaError_t attn_setup_one() {
  cudaError_t e = cudaFuncSetAttribute(k_attn_tc<F16>, cudaFuncAttributeMaxDynamicSharedMemorySize, kAttnSmem);
  if (e == cudaSuccess) e = cudaFuncSetAttribute(k_attn_tc<F16>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  return e;
}

cudaError_t attn_setup() {
  cudaError_t e = attn_setup_one<false>();
  return e == cudaSuccess ? attn_setup_one<true>() : e;
}

int attn_splits(Model& m, int ctx_hint, int T) {
  const auto& c = m.cfg;
  const int npc = attn_nodes_per_block(c.n_q_heads / c.n_kv_heads);
  const int pairs = c.n_kv_heads * ((T + npc - 1) / npc);
  const int tiles = (ctx_hint + T + kAttnKeys - 1) / kAttnKeys;
  // the most splits (one cluster of them per row block and kv head) such that
  // every cluster is resident at once -- one wave -- and no block is without a tile
  for (int sp = kMaxSplits; sp >= 1; --sp) {
    if (sp > tiles || pairs * sp > m.num_sms) continue;
    if (attn_max_clusters(sp) >= pairs) return sp;
  }
  return 1;
}

cudaError_t launch_attention(Model& m, int layer, const void* kc, const void* vc, int capacity, int ctx, int T,
                             cudaStream_t st) {
  const auto& c = m.cfg;
  if (c.dtype != OOS_DTYPE_BF16) {
    return launch(m.pdl, k_attn_f32, dim3(T, c.n_q_heads), dim3(128), 0, st, (const float*)m.ws.q, (const float*)kc,
                  (const float*)vc, (const unsigned long long*)m.ws.anc, T, c.n_q_heads, c.n_kv_heads, c.head_dim,
                  (const int32_t*)m.ws.ctx, 1.0f / sqrtf((float)c.head_dim), (float*)m.ws.attn);
  }
  AttnArgs a;
  memset(&a, 0, sizeof(a));
  // this layer's cache over its whole capacity, (d, kv head, slot); encoded
  // again only when the cache buffers change
  {
    if ((int)m.kv_maps.size() != c.n_layers) m.kv_maps.assign(c.n_layers, Model::KvMaps());
    Model::KvMaps& km = m.kv_maps[layer];
    if (km.k != kc || km.v != vc || km.extent != capacity) {
      const uint64_t dims[3] = {(uint64_t)kAttnD, (uint64_t)c.n_kv_heads, (uint64_t)capacity};
      const uint64_t strides[2] = {(uint64_t)kAttnD * 2, (uint64_t)c.n_kv_heads * kAttnD * 2};
      const uint32_t box[3] = {64, 1, (uint32_t)kAttnKeys};
      if (!encode_bf16_map(&km.kmap, kc, 3, dims, strides, box, c.kv_f16 != 0) ||
          !encode_bf16_map(&km.vmap, vc, 3, dims, strides, box, c.kv_f16 != 0)) {
        km.k = km.v = nullptr;
        return cudaErrorInvalidValue;
      }
      km.k = kc;
      km.v = vc;
      km.extent = capacity;
    }
    a.kmap = km.kmap;
    a.vmap = km.vmap;
  }
  a.qhi = m.qmap_hi;
  a.qlo = m.qmap_lo;
  a.anc = m.ws.anc;
  a.ctx_dev = m.ws.ctx;
  a.T = T;
  a.nq = c.n_q_heads;
  a.group = c.n_q_heads / c.n_kv_heads;
  a.npc = attn_nodes_per_block(a.group);
  const int RB = (T + a.npc - 1) / a.npc;
  a.splits = attn_splits(m, ctx, T);
  a.scale_log2 = 1.4426950408889634f / sqrtf((float)kAttnD);
  a.out = (__nv_bfloat16*)m.ws.attn;
  a.out_lo_off = (size_t)kMaxT * c.n_q_heads * kAttnD;
  a.status = m.ws.status;

  cudaLaunchConfig_t lc = {};
  lc.gridDim = dim3(RB, c.n_kv_heads, a.splits);
  lc.blockDim = dim3(kAttnThreads);
  lc.dynamicSmemBytes = (size_t)kAttnSmem;
  lc.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 1;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = a.splits;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  lc.attrs = attr;
  lc.numAttrs = m.pdl ? 2 : 1;
  return c.kv_f16 ? cudaLaunchKernelEx(&lc, k_attn_tc<true>, a) : cudaLaunchKernelEx(&lc, k_attn_tc<false>, a);
}

}  // namespace oos

#ifdef OOS_TIMELINE
// timeline accessors (the OOS_TIMELINE library only)
extern "C" int oos_timeline_attn_read(void* out, size_t bytes) {
  return cudaMemcpyFromSymbol(out, oos::g_tl_attn, bytes < sizeof(oos::g_tl_attn) ? bytes : sizeof(oos::g_tl_attn)) ==
                 cudaSuccess
             ? 0
             : OOS_ECUDA;
}
extern "C" int oos_timeline_attn_clear() {
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, oos::g_tl_attn) != cudaSuccess) return OOS_ECUDA;
  return cudaMemset(p, 0, sizeof(oos::g_tl_attn)) == cudaSuccess ? 0 : OOS_ECUDA;
}
#endif
