// Device helpers shared by the verify-step kernels (sm_103a).
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#define OOS_DEV __device__ __forceinline__

namespace oos {

// ---- device status word bits (reset by the first kernel of every verify)
enum : uint32_t {
  ST_TREE = 1u,      // parent[] is not parents-first / token out of range
  ST_TIMEOUT = 2u,   // a pipeline wait gave up
};

// Default limit of every pipeline wait in these kernels (nanoseconds of
// %globaltimer).  The limit in force is a per-handle value kept in the step's
// status block (words kStatusWaitLimit, +1: a 64-bit count of nanoseconds),
// set to this default by oos_model_create; waits that only drain a CTA's own
// copies or MMAs after an abort always use the default.
constexpr unsigned long long kWaitLimitNs = 2000000000ull;
constexpr int kStatusWaitLimit = 8;
OOS_DEV unsigned long long wait_limit(const uint32_t* status) {
  return *reinterpret_cast<const volatile unsigned long long*>(status + kStatusWaitLimit);
}

OOS_DEV unsigned long long globaltimer() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// ---- element conversions
OOS_DEV float to_f32(float v) { return v; }
OOS_DEV float to_f32(__nv_bfloat16 v) { return __bfloat162float(v); }
template <typename T> OOS_DEV T from_f32(float v);
template <> OOS_DEV float from_f32<float>(float v) { return v; }
template <> OOS_DEV __nv_bfloat16 from_f32<__nv_bfloat16>(float v) { return __float2bfloat16_rn(v); }

// GEMM activations of the bf16 path are stored as a pair hi = bf16(v),
// lo = bf16(v - hi) (lo at element offset lo_off): the tensor cores see v to
// about 16 mantissa bits while the weights stay bf16.  fp32 models store v.
OOS_DEV void store_act(float* p, size_t i, size_t lo_off, float v) { p[i] = v; }
OOS_DEV void store_act(__nv_bfloat16* p, size_t i, size_t lo_off, float v) {
  const __nv_bfloat16 hi = __float2bfloat16_rn(v);
  p[i] = hi;
  p[i + lo_off] = __float2bfloat16_rn(v - __bfloat162float(hi));
}

OOS_DEV void store_act4(__nv_bfloat16* p, size_t i, size_t lo_off, float4 v) {
  const float a[4] = {v.x, v.y, v.z, v.w};
  __nv_bfloat16 hi[4], lo[4];
#pragma unroll
  for (int c = 0; c < 4; ++c) {
    hi[c] = __float2bfloat16_rn(a[c]);
    lo[c] = __float2bfloat16_rn(a[c] - __bfloat162float(hi[c]));
  }
  *reinterpret_cast<uint2*>(p + i) = *reinterpret_cast<const uint2*>(hi);
  *reinterpret_cast<uint2*>(p + i + lo_off) = *reinterpret_cast<const uint2*>(lo);
}

// The same split into IEEE binary16 halves (hi = fp16(v), lo = fp16(v - hi)):
// the query layout of a model whose KV cache is binary16, so that the
// attention products multiply f16 by f16.
OOS_DEV void store_act4_h(__half* p, size_t i, size_t lo_off, float4 v) {
  const float a[4] = {v.x, v.y, v.z, v.w};
  __half hi[4], lo[4];
#pragma unroll
  for (int c = 0; c < 4; ++c) {
    hi[c] = __float2half_rn(a[c]);
    lo[c] = __float2half_rn(a[c] - __half2float(hi[c]));
  }
  *reinterpret_cast<uint2*>(p + i) = *reinterpret_cast<const uint2*>(hi);
  *reinterpret_cast<uint2*>(p + i + lo_off) = *reinterpret_cast<const uint2*>(lo);
}

// ---- block reductions (deterministic order)
OOS_DEV float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
OOS_DEV float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
// sum over the block; `red` is shared scratch of >= 32 floats; all threads get the result
OOS_DEV float block_sum(float v, float* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  v = warp_sum(v);
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  float s = 0.f;
  for (int i = 0; i < nw; ++i) s += red[i];
  return s;
}
OOS_DEV float block_max(float v, float* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  v = warp_max(v);
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  float s = -INFINITY;
  for (int i = 0; i < nw; ++i) s = fmaxf(s, red[i]);
  return s;
}

// ---- programmatic dependent launch
OOS_DEV void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
OOS_DEV void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// ---- shared-memory addresses and mbarriers
OOS_DEV uint32_t smem_addr(const void* p) { return static_cast<uint32_t>(__cvta_generic_to_shared(p)); }

OOS_DEV void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}
OOS_DEV void mbar_fence_init() { asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory"); }
OOS_DEV void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
               : "memory");
}
OOS_DEV void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}
OOS_DEV bool mbar_test(uint32_t addr, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(addr), "r"(parity)
      : "memory");
  return ok != 0;
}
// Same test, but a thread whose phase is not complete yet is suspended (issue
// slots go to the warps with work) until it completes or `hint_ns` pass.
OOS_DEV bool mbar_test_sleep(uint32_t addr, uint32_t parity, uint32_t hint_ns) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(addr), "r"(parity), "r"(hint_ns)
      : "memory");
  return ok != 0;
}
// First wait of the step to exceed its limit: status[1] = site code, [2] = phase,
// [3] = unit or tile, [4] = CTA, [5] = block-local detail (first writer wins).
OOS_DEV void record_timeout(uint32_t* status, uint32_t site, int phase, long long unit, int detail) {
  if (atomicCAS(status + 1, 0u, site) == 0u) {
    status[2] = (uint32_t)phase;
    status[3] = (uint32_t)unit;
    status[4] = blockIdx.x;
    status[5] = (uint32_t)detail;
  }
}

// Wait for the phase with `parity` to complete.  Gives up after the handle's
// wait limit or when *abort becomes nonzero (another role gave up); returns
// false then and records ST_TIMEOUT in *status (only for a genuine timeout).
// Between checks of the abort flag the thread sleeps on the barrier (at most
// 20 us, and at most the limit, at a time).
OOS_DEV bool mbar_wait(uint64_t* bar, uint32_t parity, volatile int* abort, uint32_t* status) {
  const uint32_t addr = smem_addr(bar);
  if (mbar_test(addr, parity)) return true;
  const unsigned long long t0 = globaltimer();
  const unsigned long long limit = wait_limit(status);
  const uint32_t hint = limit < 20000ull ? (uint32_t)limit : 20000u;
  while (true) {
    if (mbar_test_sleep(addr, parity, hint)) return true;
    if (*abort) return false;
    if (globaltimer() - t0 > limit) {
      *abort = 1;
      atomicOr(status, ST_TIMEOUT);
      return false;
    }
  }
}

// ---- TMA (tiled tensor copies, global -> shared)
OOS_DEV uint64_t policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
OOS_DEV uint64_t policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}
OOS_DEV void tma_prefetch_desc(const void* tmap) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(tmap)) : "memory");
}
// 2-D tile load; x = innermost coordinate (elements), y = row.  x*2 bytes must
// be a multiple of 16 (callers pass multiples of 64 bf16 elements).
OOS_DEV void tma_load_2d(void* smem_dst, const void* tmap, uint64_t* bar, int x, int y, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(smem_addr(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(x), "r"(y), "r"(smem_addr(bar)), "l"(policy)
      : "memory");
}

// 3-D / 4-D tile loads (coordinates innermost first; x * 2 bytes a multiple of 16)
OOS_DEV void tma_load_3d(void* smem_dst, const void* tmap, uint64_t* bar, int x, int y, int z, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3, %4}], [%5], %6;" ::"r"(smem_addr(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(x), "r"(y), "r"(z), "r"(smem_addr(bar)), "l"(policy)
      : "memory");
}
OOS_DEV void tma_load_4d(void* smem_dst, const void* tmap, uint64_t* bar, int x, int y, int z, int w,
                         uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3, %4, %5}], [%6], %7;" ::"r"(smem_addr(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(x), "r"(y), "r"(z), "r"(w), "r"(smem_addr(bar)), "l"(policy)
      : "memory");
}

// ---- tcgen05 (5th-generation tensor cores, accumulators in TMEM)
OOS_DEV void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
OOS_DEV void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// whole warp: allocate `ncols` TMEM columns, base address written to *slot
OOS_DEV void tmem_alloc(uint32_t* slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(slot)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
OOS_DEV void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

// Shared-memory matrix descriptor, K-major operand staged by TMA with the
// 128-byte swizzle: rows of 128 bytes, 8-row (1024-byte) swizzle atoms.
//   bits  0-13 start address >> 4     bits 16-29 leading byte offset >> 4 (unused here)
//   bits 32-45 stride byte offset >> 4 (1024: next 8-row group)
//   bits 46-48 fixed 0b001            bits 49-51 base offset (0: atoms 1024-aligned)
//   bit  52    LBO mode (0)           bits 61-63 swizzle (2 = 128-byte)
OOS_DEV uint64_t smem_desc_sw128(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)1 << 16;
  d |= (uint64_t)(1024u >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

// Instruction descriptor of tcgen05.mma.kind::f16 with bf16 A and B, fp32 D,
// both operands K-major, shape M x N.
//   bits 4-5 D format (1 = f32), 7-9 A format (1 = bf16), 10-12 B format (1 = bf16),
//   15/16 A/B major (0 = K), 17-22 N >> 3, 24-28 M >> 4
__host__ __device__ constexpr uint32_t idesc_bf16_f32(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

// Same for f16 A and B (format 0 in both fields), fp32 D.
__host__ __device__ constexpr uint32_t idesc_f16_f32(int M, int N) {
  return (1u << 4) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

// D[tmem] (+)= A[smem] * B[smem]^T, one elected thread issues
OOS_DEV void tc_mma_bf16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// arrive on *bar once all previously issued tcgen05.mma of this thread complete
OOS_DEV void tc_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                   smem_addr(bar))
               : "memory");
}
// 32 lanes x 32 bit, 16 consecutive columns per thread
OOS_DEV void tmem_ld16(uint32_t taddr, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// Same load without its wait: the caller issues several, then tmem_wait_ld
// and reg_fence over every register loaded (the empty statements make each
// later use of those registers depend on the wait).
OOS_DEV void tmem_ld16_nowait(uint32_t taddr, float (&v)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=f"(v[0]), "=f"(v[1]), "=f"(v[2]), "=f"(v[3]), "=f"(v[4]), "=f"(v[5]), "=f"(v[6]), "=f"(v[7]),
        "=f"(v[8]), "=f"(v[9]), "=f"(v[10]), "=f"(v[11]), "=f"(v[12]), "=f"(v[13]), "=f"(v[14]), "=f"(v[15])
      : "r"(taddr));
}
OOS_DEV void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
template <int N>
OOS_DEV void reg_fence(float (&v)[N]) {
#pragma unroll
  for (int i = 0; i < N; ++i) asm volatile("" : "+f"(v[i]));
}

}  // namespace oos
