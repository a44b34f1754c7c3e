// Weight-streaming GEMMs of the verify step.
//
// bf16 path (tcgen05): D[f, t] = sum_k W[f, k] * X[t, k] with the weight rows
// f in the MMA's M = 128 slot and the T tree nodes in N ("swap-AB": T <= 128
// is far too small for M).  Weights are the only large operand; each is read
// from HBM exactly once per step.  Per CTA: one TMA producer thread streams
// 128 x 64 weight tiles and the matching 64-wide slice of X through an
// S-stage shared-memory ring; one thread issues tcgen05.mma into a TMEM
// accumulator (two buffers, so the epilogue of one tile overlaps the MMAs of
// the next); four epilogue warps drain TMEM with tcgen05.ld.
//   MODE_PARTIAL: stream-K over (tile, k-block) units, fp32 partial tiles out.
//   MODE_ARGMAX : LM head, whole tiles round-robin, per-node running
//                 (max, argmax, second max) -- logits never reach memory.
//
// fp32 path: CUDA-core warp-per-row GEMV kernels (small models only).
#include <string.h>

#include "common.cuh"
#include "internal.h"

namespace oos {

enum { MODE_PARTIAL = 0, MODE_ARGMAX = 1 };

struct GemmArgs {
  int seg_tiles[3];   // cumulative tile counts per weight segment
  int n_tiles, kbt, total;
  int N;              // output rows (features / vocab)
  int T;              // valid columns (tree nodes)
  float* part;        // MODE_PARTIAL: [slice][kMaxT][N]
  float* am_v1;       // MODE_ARGMAX: [cta][kMaxT]
  int32_t* am_i;
  float* am_v2;
  uint32_t* status;
};

template <int BN>
struct TcCfg {
  static constexpr int A_BYTES = kTile * kBK * 2;              // 16 KB weight tile
  static constexpr int B_BYTES = BN * kBK * 2;                 // one activation half (hi or lo)
  static constexpr int STAGE = A_BYTES + 2 * B_BYTES;
  static constexpr int S_RAW = (200 * 1024) / STAGE;
  static constexpr int S = S_RAW > 8 ? 8 : S_RAW;
  static constexpr int NCOLS = (2 * BN) < 32 ? 32 : 2 * BN;    // two accumulators, power of two
  static constexpr int BAR_BYTES = 1024;
  static constexpr int RED_BYTES = 4 * BN * 12 + BN * 12;      // argmax cross-warp scratch + running state
  static constexpr int SMEM = 1024 /*align slack*/ + S * STAGE + BAR_BYTES + RED_BYTES;
};

struct Top2s {
  float v1;
  int i1;
  float v2;
};
OOS_DEV Top2s t2_merge(Top2s a, Top2s b) {
  Top2s r;
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

template <int BN, int MODE>
__global__ void __launch_bounds__(192, 1)
    k_gemm_tc(const __grid_constant__ CUtensorMap wm0, const __grid_constant__ CUtensorMap wm1,
              const __grid_constant__ CUtensorMap wm2, const __grid_constant__ CUtensorMap am, GemmArgs a) {
  using C = TcCfg<BN>;
  constexpr int S = C::S;
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  unsigned char* sA = smem;
  unsigned char* sB = smem + S * C::A_BYTES;      // [stage][hi|lo][BN rows x 128 B]
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S * C::STAGE);
  uint64_t* empty = full + S;
  uint64_t* accf = empty + S;
  uint64_t* acce = accf + 2;
  uint64_t* drain = acce + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  Top2s* red = reinterpret_cast<Top2s*>(smem + S * C::STAGE + C::BAR_BYTES);   // [4][BN]
  Top2s* run = red + 4 * BN;                                                    // [BN]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = gridDim.x, cta = blockIdx.x;

  // this CTA's work: units [u0, u1) (stream-K) or tiles cta, cta+G, ... (argmax)
  long long u0, u1;
  if (MODE == MODE_PARTIAL) {
    u0 = (long long)cta * a.total / G;
    u1 = (long long)(cta + 1) * a.total / G;
  } else {
    const int my_tiles = cta < a.n_tiles ? (a.n_tiles - cta + G - 1) / G : 0;
    u0 = 0;
    u1 = (long long)my_tiles * a.kbt;
  }
  const int n_units = (int)(u1 - u0);
  auto unit_tile = [&](int j, int& tile, int& kb) {
    if (MODE == MODE_PARTIAL) {
      const long long u = u0 + j;
      tile = (int)(u / a.kbt);
      kb = (int)(u % a.kbt);
    } else {
      tile = cta + (j / a.kbt) * G;
      kb = j % a.kbt;
    }
  };

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&accf[b], 1);
      mbar_init(&acce[b], 4);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    mbar_fence_init();
  }
  if (warp == 2) tmem_alloc(tmem_slot, C::NCOLS);
  if (MODE == MODE_ARGMAX && threadIdx.x >= 64) {
    for (int e = threadIdx.x - 64; e < BN; e += 128) run[e] = Top2s{-INFINITY, 0x7fffffff, -INFINITY};
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      tma_prefetch_desc(&wm0);
      tma_prefetch_desc(&am);
      const uint64_t pol_w = policy_evict_first();
      const uint64_t pol_a = policy_evict_last();
      auto load_w = [&](int j, int stage) {
        int tile, kb;
        unit_tile(j, tile, kb);
        const CUtensorMap* wm = &wm0;
        int row = tile * kTile;
        if (tile >= a.seg_tiles[0]) {
          if (tile >= a.seg_tiles[1]) {
            wm = &wm2;
            row = (tile - a.seg_tiles[1]) * kTile;
          } else {
            wm = &wm1;
            row = (tile - a.seg_tiles[0]) * kTile;
          }
        }
        tma_load_2d(sA + stage * C::A_BYTES, wm, &full[stage], kb * kBK, row, pol_w);
      };
      auto load_x = [&](int j, int stage) {
        int tile, kb;
        unit_tile(j, tile, kb);
        unsigned char* dst = sB + stage * 2 * C::B_BYTES;
        tma_load_2d(dst, &am, &full[stage], kb * kBK, 0, pol_a);                   // hi rows
        tma_load_2d(dst + C::B_BYTES, &am, &full[stage], kb * kBK, kMaxT, pol_a);  // lo rows
      };
      // weights do not depend on the previous kernel: start streaming them
      // before waiting for it (programmatic dependent launch)
      const int n_pre = n_units < S ? n_units : S;
      for (int j = 0; j < n_pre; ++j) {
        mbar_arrive_expect_tx(&full[j], C::STAGE);
        load_w(j, j);
      }
      pdl_wait();
      for (int j = 0; j < n_pre; ++j) load_x(j, j);
      int stage = n_pre % S;
      uint32_t phase = (n_pre == S) ? 1u : 0u;
      int issued = n_pre;
      for (int j = n_pre; j < n_units; ++j) {
        if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, a.status)) break;
        mbar_arrive_expect_tx(&full[stage], C::STAGE);
        load_w(j, stage);
        load_x(j, stage);
        ++issued;
        if (++stage == S) {
          stage = 0;
          phase ^= 1u;
        }
      }
      if (*abort_flag) {
        // let this CTA's copies in flight land before the CTA exits
        const int first = issued - S > 0 ? issued - S : 0;
        for (int j = first; j < issued; ++j) {
          const unsigned long long t0 = globaltimer();
          while (!mbar_test(smem_addr(&full[j % S]), (uint32_t)((j / S) & 1)) && globaltimer() - t0 < kWaitLimitNs) {
          }
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    pdl_wait();
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(kTile, BN);
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_use[2] = {0, 0};
      int j = 0;
      bool ok = true;
      while (j < n_units && ok) {
        int tile, kb;
        unit_tile(j, tile, kb);
        int seg_end = j + (a.kbt - kb);       // units of this tile owned here
        if (seg_end > n_units) seg_end = n_units;
        if (!mbar_wait(&acce[acc], (acc_use[acc] & 1u) ^ 1u, abort_flag, a.status)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * BN);
        for (int jj = j; jj < seg_end; ++jj) {
          if (!mbar_wait(&full[stage], phase, abort_flag, a.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t ad = smem_desc_sw128(smem_addr(sA + stage * C::A_BYTES));
          const uint64_t bh = smem_desc_sw128(smem_addr(sB + stage * 2 * C::B_BYTES));
          const uint64_t bl = smem_desc_sw128(smem_addr(sB + stage * 2 * C::B_BYTES + C::B_BYTES));
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k) {
            tc_mma_bf16(d_tmem, ad + 2 * k, bh + 2 * k, idesc, (jj > j || k > 0) ? 1u : 0u);
            tc_mma_bf16(d_tmem, ad + 2 * k, bl + 2 * k, idesc, 1u);
          }
          tc_commit(&empty[stage]);
          if (++stage == S) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        tc_commit(&accf[acc]);
        ++acc_use[acc];
        acc ^= 1;
        j = seg_end;
      }
      // all issued MMAs complete before TMEM is released
      tc_commit(drain);
      const unsigned long long t0 = globaltimer();
      while (!mbar_test(smem_addr(drain), 0) && globaltimer() - t0 < kWaitLimitNs) {
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue (warps 2..5)
    pdl_wait();
    const int q = warp & 3;               // TMEM lane quarter this warp may access
    const int row = q * 32 + lane;
    const int e = threadIdx.x - 64;       // 0..127
    int acc = 0;
    uint32_t acc_use[2] = {0, 0};
    int j = 0;
    while (j < n_units) {
      int tile, kb;
      unit_tile(j, tile, kb);
      int seg_end = j + (a.kbt - kb);
      if (seg_end > n_units) seg_end = n_units;
      if (!mbar_wait(&accf[acc], acc_use[acc] & 1u, abort_flag, a.status)) break;
      tc_fence_after();
      const uint32_t taddr = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * BN);
      const int f = tile * kTile + row;
      if (MODE == MODE_PARTIAL) {
        int c0, c1;
        StreamK sk{a.n_tiles, a.kbt, a.total, G};
        sk.contributors(tile, c0, c1);
        float* dst = a.part + (size_t)(cta - c0) * kMaxT * a.N + f;
#pragma unroll 1
        for (int cc = 0; cc < BN / 16; ++cc) {
          if (cc * 16 >= a.T) break;
          float v[16];
          tmem_ld16(taddr + cc * 16, v);
          if (f < a.N) {
#pragma unroll
            for (int i = 0; i < 16; ++i) {
              const int t = cc * 16 + i;
              if (t < a.T) dst[(size_t)t * a.N] = v[i];
            }
          }
        }
      } else {
#pragma unroll 1
        for (int cc = 0; cc < BN / 16; ++cc) {
          if (cc * 16 >= a.T) break;
          float v[16];
          tmem_ld16(taddr + cc * 16, v);
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            Top2s s{f < a.N ? v[i] : -INFINITY, f, -INFINITY};
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
              Top2s y;
              y.v1 = __shfl_xor_sync(0xffffffffu, s.v1, o);
              y.i1 = __shfl_xor_sync(0xffffffffu, s.i1, o);
              y.v2 = __shfl_xor_sync(0xffffffffu, s.v2, o);
              s = t2_merge(s, y);
            }
            if (lane == 0) red[q * BN + cc * 16 + i] = s;
          }
        }
        asm volatile("bar.sync 1, 128;" ::: "memory");
        if (e < a.T) {
          Top2s r = run[e];
#pragma unroll
          for (int w = 0; w < 4; ++w) r = t2_merge(r, red[w * BN + e]);
          run[e] = r;
        }
        asm volatile("bar.sync 1, 128;" ::: "memory");
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acce[acc]);
      ++acc_use[acc];
      acc ^= 1;
      j = seg_end;
    }
    if (MODE == MODE_ARGMAX && e < a.T) {
      const Top2s r = run[e];
      a.am_v1[(size_t)cta * kMaxT + e] = r.v1;
      a.am_i[(size_t)cta * kMaxT + e] = r.i1;
      a.am_v2[(size_t)cta * kMaxT + e] = r.v2;
    }
  }
  pdl_trigger();
  tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem_base, C::NCOLS);
  }
}

// ------------------------------------------------------------ host side
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn get_encode() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

static bool encode_2d(CUtensorMap* map, const void* ptr, int rows, int K, int box_rows) {
  EncodeTiledFn enc = get_encode();
  if (!enc) return false;
  memset(map, 0, sizeof(*map));
  cuuint64_t gdim[2] = {(cuuint64_t)K, (cuuint64_t)rows};
  cuuint64_t gstride[1] = {(cuuint64_t)K * 2};
  cuuint32_t box[2] = {(cuuint32_t)kBK, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), gdim, gstride, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool encode_weight_map(CUtensorMap* map, const void* ptr, int rows, int K) {
  return encode_2d(map, ptr, rows, K, kTile);
}
bool encode_act_map(CUtensorMap* map, const void* ptr, int K, int box_rows) {
  return encode_2d(map, ptr, 2 * kMaxT, K, box_rows);   // hi rows [0, 128), lo rows [128, 256)
}

int bn_index(int T) { return T <= 16 ? 0 : T <= 32 ? 1 : T <= 64 ? 2 : 3; }

template <int BN, int MODE>
static cudaError_t set_smem() {
  return cudaFuncSetAttribute(k_gemm_tc<BN, MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize, TcCfg<BN>::SMEM);
}

cudaError_t gemm_setup() {
  cudaError_t e = cudaSuccess;
  cudaError_t r;
#define OOS_SET(BN)                                       \
  if ((r = set_smem<BN, MODE_PARTIAL>()) != cudaSuccess) e = r; \
  if ((r = set_smem<BN, MODE_ARGMAX>()) != cudaSuccess) e = r;
  OOS_SET(16) OOS_SET(32) OOS_SET(64) OOS_SET(128)
#undef OOS_SET
  return e;
}

template <int BN, int MODE>
static cudaError_t launch_tc(Model& m, const GemmW& g, const CUtensorMap& amap, int T, int grid, GemmArgs& a,
                             cudaStream_t st) {
  const CUtensorMap& w1 = g.n_seg > 1 ? g.map[1] : g.map[0];
  const CUtensorMap& w2 = g.n_seg > 2 ? g.map[2] : g.map[0];
  return launch(m.pdl, k_gemm_tc<BN, MODE>, dim3(grid), dim3(192), (size_t)TcCfg<BN>::SMEM, st, g.map[0], w1, w2,
                amap, a);
}

template <int MODE>
static cudaError_t dispatch_tc(Model& m, const GemmW& g, const CUtensorMap& amap, int T, int grid, GemmArgs& a,
                               cudaStream_t st) {
  switch (bn_index(T)) {
    case 0: return launch_tc<16, MODE>(m, g, amap, T, grid, a, st);
    case 1: return launch_tc<32, MODE>(m, g, amap, T, grid, a, st);
    case 2: return launch_tc<64, MODE>(m, g, amap, T, grid, a, st);
    default: return launch_tc<128, MODE>(m, g, amap, T, grid, a, st);
  }
}

static GemmArgs base_args(Model& m, const GemmW& g, int T) {
  GemmArgs a;
  memset(&a, 0, sizeof(a));
  for (int s = 0; s < 3; ++s) a.seg_tiles[s] = g.seg_tiles[s < g.n_seg ? s : g.n_seg - 1];
  a.n_tiles = g.plan.n_tiles;
  a.kbt = g.plan.kbt;
  a.total = g.plan.total;
  a.N = g.N;
  a.T = T;
  a.status = m.ws.status;
  return a;
}

cudaError_t launch_gemm_tc(Model& m, const GemmW& g, const CUtensorMap& amap, int T, cudaStream_t st) {
  GemmArgs a = base_args(m, g, T);
  a.part = m.ws.part;
  return dispatch_tc<MODE_PARTIAL>(m, g, amap, T, g.plan.grid, a, st);
}

cudaError_t launch_lm_head_tc(Model& m, int T, cudaStream_t st) {
  GemmArgs a = base_args(m, m.g_lm, T);
  a.am_v1 = m.ws.lm_v1;
  a.am_i = m.ws.lm_i;
  a.am_v2 = m.ws.lm_v2;
  return dispatch_tc<MODE_ARGMAX>(m, m.g_lm, m.amap_xn[bn_index(T)], T, m.lm_grid, a, st);
}

// ------------------------------------------------------------ fp32 CUDA-core path
// One warp per output row; part[t][f] = W[f] . x[t] (a single slice).
__global__ void __launch_bounds__(128) k_gemm_f32(const float* __restrict__ w0, const float* __restrict__ w1,
                                                  const float* __restrict__ w2, int r0, int r1, int r2, int K,
                                                  const float* __restrict__ x, int T, float* __restrict__ part) {
  pdl_wait();
  const int N = r0 + r1 + r2;
  const int f = blockIdx.x * 4 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (f < N) {
    const float* w = f < r0 ? w0 + (size_t)f * K : f < r0 + r1 ? w1 + (size_t)(f - r0) * K : w2 + (size_t)(f - r0 - r1) * K;
    for (int t = 0; t < T; ++t) {
      const float* xr = x + (size_t)t * K;
      float acc = 0.f;
      for (int k = lane; k < K; k += 32) acc += w[k] * xr[k];
      acc = warp_sum(acc);
      if (lane == 0) part[(size_t)t * N + f] = acc;
    }
  }
  pdl_trigger();
}

cudaError_t launch_gemm_f32(Model& m, const void* w0, const void* w1, const void* w2, int rows0, int rows1, int rows2,
                            int K, const void* x, int T, cudaStream_t st) {
  const int N = rows0 + rows1 + rows2;
  return launch(m.pdl, k_gemm_f32, dim3((N + 3) / 4), dim3(128), 0, st, (const float*)w0, (const float*)w1,
                (const float*)w2, rows0, rows1, rows2, K, (const float*)x, T, m.ws.part);
}

// LM head, fp32: block b scans vocab rows [b*rows, (b+1)*rows); warp w keeps a
// running top-2 per node over its rows; warps merge in order at the end.
__global__ void __launch_bounds__(128) k_lm_head_f32(const float* __restrict__ W, int V, int H, int rows_per_block,
                                                     const float* __restrict__ x, int T, float* am_v1, int32_t* am_i,
                                                     float* am_v2) {
  __shared__ Top2s st[4][kMaxT];
  pdl_wait();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int t = lane; t < T; t += 32) st[warp][t] = Top2s{-INFINITY, 0x7fffffff, -INFINITY};
  const int r_begin = blockIdx.x * rows_per_block;
  const int r_end = min(V, r_begin + rows_per_block);
  for (int r = r_begin + warp; r < r_end; r += 4) {
    const float* w = W + (size_t)r * H;
    for (int t = 0; t < T; ++t) {
      const float* xr = x + (size_t)t * H;
      float acc = 0.f;
      for (int k = lane; k < H; k += 32) acc += w[k] * xr[k];
      acc = warp_sum(acc);
      if (lane == 0) st[warp][t] = t2_merge(st[warp][t], Top2s{acc, r, -INFINITY});
    }
  }
  __syncthreads();
  for (int t = threadIdx.x; t < T; t += blockDim.x) {
    Top2s r = st[0][t];
    for (int w = 1; w < 4; ++w) r = t2_merge(r, st[w][t]);
    am_v1[(size_t)blockIdx.x * kMaxT + t] = r.v1;
    am_i[(size_t)blockIdx.x * kMaxT + t] = r.i1;
    am_v2[(size_t)blockIdx.x * kMaxT + t] = r.v2;
  }
  pdl_trigger();
}

cudaError_t launch_lm_head_f32(Model& m, int T, cudaStream_t st) {
  const int V = m.cfg.vocab;
  const int rows = (V + m.lm_grid - 1) / m.lm_grid;
  return launch(m.pdl, k_lm_head_f32, dim3(m.lm_grid), dim3(128), 0, st, (const float*)m.w.lm_head, V, m.cfg.hidden,
                rows, (const float*)m.ws.xn, T, m.ws.lm_v1, m.ws.lm_i, m.ws.lm_v2);
}

}  // namespace oos
