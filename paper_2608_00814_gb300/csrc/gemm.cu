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
// The layer's elementwise steps run in the GEMM epilogues (see below); the LM
// head keeps a per-node running (max, argmax, second max) so logits never
// reach memory.
//
// fp32 path: CUDA-core warp-per-row GEMV kernels (small models only).
#include <string.h>

#include "common.cuh"
#include "internal.h"

// Step timeline (built only with -DOOS_TIMELINE, see timeline.py): per GEMM
// launch of a step and per CTA, the globaltimer at entry (0), at the end of the
// dependency wait (1), when the last accumulator is ready (2), at the last
// arrival count (4), when the finishing may start (5) and at exit (3).  A
// launch's slot comes from its arrival-counter block, one per (layer, GEMM).
#ifdef OOS_TIMELINE
namespace oos {
__device__ unsigned long long g_tl_gemm[1024][160][6];
}
#define TL_GEMM(ev)                                                                                   \
  do {                                                                                                \
    if (!ARGMAX && a.cnt && blockIdx.x < 160)                                                        \
      oos::g_tl_gemm[((uintptr_t)a.cnt >> 10) & 1023][blockIdx.x][ev] = oos::globaltimer();          \
  } while (0)
#else
#define TL_GEMM(ev) \
  do {              \
  } while (0)
#endif

namespace oos {

// Epilogues fused into the weight GEMMs (bf16 path).  Stream-K leaves a tile's
// reduction split over up to a few CTAs: each writes its fp32 partial tile,
// and the LAST contributor to arrive (a per-tile arrival counter) adds the
// slices in slice order -- a fixed order, so results are deterministic -- and
// applies the layer's elementwise step to the finished tile:
//   EPI_QKV   : input RMSNorm scale, bias, per-head q/k RMSNorm, RoPE at
//               ctx + depth; q (hi/lo bf16) to the query buffer, k/v to cache
//               slot ctx + t.
//   EPI_RESID : x += W.a (O- and down-projections), then y = g (.) x for the
//               next RMSNorm (hi/lo bf16) and per-tile sums of x^2.
//   EPI_SILU  : gate and up tiles are interleaved (tile 2i = gate rows of
//               block i, 2i+1 = up rows); act = silu(r g) * (r u).
//   EPI_ARGMAX: LM head -- whole tiles round-robin, logits scaled by the final
//               RMSNorm factor and folded into a per-node running top-2.
// RMSNorm is split across kernels by linearity: a producer stores y = g (.) x
// and sum(x^2) per 128-feature chunk; the consumer GEMM computes W.y and
// multiplies column t by r_t = rsqrt(sum x_t^2 / H + eps) in its epilogue.
enum { EPI_QKV = 0, EPI_RESID = 1, EPI_SILU = 2, EPI_ARGMAX = 3 };

// A work tile is SUB weight subtiles of 128 rows (the MMA's M) that share every
// staged activation slice.  The gate/up GEMM and the LM head use SUB = 2 (per
// weight byte half the activation traffic, more weight bytes in flight, and
// gate + up rows of one block in one CTA); the smaller QKV, O and down GEMMs
// use SUB = 1 so each tile has fewer stream-K contributors.  Subtile s of work
// tile w is the 128-row tile SUB*w + s of the stacked weight.
template <int EPI>
struct SubOf {
  static constexpr int v = (EPI == 2 || EPI == 3) ? 2 : 1;
};

struct GemmArgs {
  int seg_tiles[3];   // cumulative 128-row tile counts per weight segment
  int interleave2;    // 128-row tile 2i -> segment 0 block i, tile 2i+1 -> segment 1 block i
  int n_tiles;        // 128-row tiles of the stacked weight
  int n_work, kbt, total;   // work tiles (SUB subtiles each), k-blocks per tile, n_work * kbt
  int N;              // output rows (features / vocab) of the stacked weight
  int T;              // valid columns (tree nodes)
  float* part;        // partial tiles [slice][kMaxT][n_work * SUB * 128]
  int* cnt;           // arrival counter per work tile (zeroed at every step start)
  uint32_t* status;
  // RMSNorm scale of the GEMM input (EPI_QKV, EPI_SILU, EPI_ARGMAX)
  const float* ss_in;   // [chunk][kMaxT]
  int ss_chunks;
  float inv_dim, eps;
  // EPI_QKV
  int nq, nkv;
  const __nv_bfloat16 *bq, *bk, *bv, *gq, *gk;
  const float2* rope;   // [kMaxT][64] (cos, sin) of the step's positions
  __nv_bfloat16 *q_out, *kc, *vc;
  const int32_t* ctx;   // committed length of the step (device; K/V of node t go to slot *ctx + t)
  int kv_f16;           // the KV cache (and so q) are binary16 instead of bf16
  // EPI_RESID
  float* x;
  const __nv_bfloat16* gain;
  __nv_bfloat16* y_out;
  float* ss_out;
  // EPI_SILU
  __nv_bfloat16* act_out;
  int I;
  // EPI_ARGMAX
  float* am_v1;
  int32_t* am_i;
  float* am_v2;
};

template <int BN, int kSub>
struct TcCfg {
  static constexpr int A_BYTES = kTile * kBK * 2;              // 16 KB per 128-row weight subtile
  static constexpr int B_BYTES = BN * kBK * 2;                 // one activation half (hi or lo)
  static constexpr int STAGE = kSub * A_BYTES + 2 * B_BYTES;
  static constexpr int BAR_BYTES = 256;
  static constexpr int EPI_BYTES = kMaxT * 4 + 64;             // input RMSNorm factors, flags
  static constexpr int RED_BYTES = 4 * BN * 12 + BN * 12;      // argmax cross-warp scratch + running state
  static constexpr int FIXED = 1024 /*align slack*/ + BAR_BYTES + EPI_BYTES + RED_BYTES;
  static constexpr int S_RAW = (227 * 1024 - FIXED) / STAGE;
  static constexpr int S = S_RAW > 8 ? 8 : S_RAW;
  // The hi and lo activation halves sit in one slot, hi rows then lo rows, so
  // one MMA with N = 2 BN multiplies both ("paired": half the MMAs, the weight
  // subtile read from shared memory once); the accumulator then holds the hi
  // products in columns [0, BN) and the lo products in [BN, 2 BN).  Paired
  // when two buffers of kSub such accumulators fit the 512 TMEM columns.
  static constexpr bool PAIRED = 2 * kSub * 2 * BN <= 512;
  static constexpr int SUB_COLS = PAIRED ? 2 * BN : BN;                      // accumulator columns per subtile
  static constexpr int NCOLS = (2 * kSub * SUB_COLS) < 32 ? 32 : 2 * kSub * SUB_COLS;   // 2 buffers
  static constexpr int SMEM = FIXED + S * STAGE;
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

OOS_DEV void epi_bar() { asm volatile("bar.sync 1, 128;" ::: "memory"); }


// Finishing a subtile: warp w of the four epilogue warps owns token rows
// t = t0 + 4k + w, lane l owns the four features 4l..4l+3 of the subtile, so a
// token's 128 features sit in one warp (RMSNorm sums, q/k norm and the RoPE
// pair exchange are warp shuffles) and every slice load is a coalesced float4.
// All loads of a pass are issued before any result is stored.
constexpr int kFinRows = 4;    // token rows per warp per pass (16 tokens per pass)

OOS_DEV float4 f4_add(float4 a, float4 b) { return make_float4(a.x + b.x, a.y + b.y, a.z + b.z, a.w + b.w); }
OOS_DEV float4 f4_ldcg(const float* p) { return __ldcg(reinterpret_cast<const float4*>(p)); }

// Where a finishing pass reads the partial sums of output (token t, feature f)
// from: partial s of nc, the stream-K slices in global memory,
// [slice][kMaxT][n_part] (feature f of the stacked weight).
struct GSrc {
  const float* p;
  size_t slice;
  int ld;
  OOS_DEV float4 ld4(int s, int t, int f) const { return f4_ldcg(p + (size_t)s * slice + (size_t)t * ld + f); }
};

// acc[k] = (init ? init row : 0) + sum over nc slices of the partial tile rows,
// rows t = t0 + nw k + w below T (the end of the token range; w is this warp's
// index among the nw warps finishing the tile).  Slices are
// fetched BATCH at a time -- every load of a group is issued before any is
// added -- and added in slice order, so the sum is the same for every finisher.
template <int R, int BATCH, typename Src>
OOS_DEV void load_tile_rows(float4 (&acc)[R], const Src& src, int nc, int col, int t0, int T,
                            const float* __restrict__ init, int init_ld, int init_col, int w, int nw) {
#pragma unroll
  for (int k = 0; k < R; ++k) {
    const int t = t0 + nw * k + w;
    acc[k] = (init && t < T) ? *reinterpret_cast<const float4*>(init + (size_t)t * init_ld + init_col)
                             : make_float4(0.f, 0.f, 0.f, 0.f);
  }
  for (int s0 = 0; s0 < nc; s0 += BATCH) {
    float4 v[BATCH][R];
#pragma unroll
    for (int q = 0; q < BATCH; ++q) {
#pragma unroll
      for (int k = 0; k < R; ++k) {
        const int t = t0 + nw * k + w;
        v[q][k] = (s0 + q < nc && t < T) ? src.ld4(s0 + q, t, col) : make_float4(0.f, 0.f, 0.f, 0.f);
      }
    }
#pragma unroll
    for (int q = 0; q < BATCH; ++q)
#pragma unroll
      for (int k = 0; k < R; ++k) acc[k] = f4_add(acc[k], v[q][k]);
  }
}

// gate (col) and up (col + up_off) rows of a SwiGLU pair, two slices per batch
template <int R, typename Src>
OOS_DEV void load_pair_rows(float4 (&g)[R], float4 (&u)[R], const Src& src, int nc, int col, int up_off, int t0,
                            int T, int w, int nw) {
#pragma unroll
  for (int k = 0; k < R; ++k) g[k] = u[k] = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int s0 = 0; s0 < nc; s0 += 2) {
    float4 vg[2][R], vu[2][R];
#pragma unroll
    for (int q = 0; q < 2; ++q) {
#pragma unroll
      for (int k = 0; k < R; ++k) {
        const int t = t0 + nw * k + w;
        const bool ok = s0 + q < nc && t < T;
        vg[q][k] = ok ? src.ld4(s0 + q, t, col) : make_float4(0.f, 0.f, 0.f, 0.f);
        vu[q][k] = ok ? src.ld4(s0 + q, t, col + up_off) : make_float4(0.f, 0.f, 0.f, 0.f);
      }
    }
#pragma unroll
    for (int q = 0; q < 2; ++q)
#pragma unroll
      for (int k = 0; k < R; ++k) {
        g[k] = f4_add(g[k], vg[q][k]);
        u[k] = f4_add(u[k], vu[q][k]);
      }
  }
}

OOS_DEV float4 bf16x4(const __nv_bfloat16* p) {
  const uint2 u = *reinterpret_cast<const uint2*>(p);
  const __nv_bfloat16* h = reinterpret_cast<const __nv_bfloat16*>(&u);
  return make_float4(__bfloat162float(h[0]), __bfloat162float(h[1]), __bfloat162float(h[2]), __bfloat162float(h[3]));
}

// EPI_RESID on 128-row tile `tile`, tokens [tb, te), by warp w of nw: x += W.a;
// y = g (.) x; per-tile sums of x^2
template <typename Src>
OOS_DEV void finish_resid(const GemmArgs& a, const Src& src, int tile, int nc, int tb, int te, int w, int nw) {
  const int l = threadIdx.x & 31;
  const int f = tile * kTile + 4 * l;
  const float4 g = bf16x4(a.gain + f);
  for (int t0 = tb; t0 < te; t0 += nw * kFinRows) {
    float4 acc[kFinRows];
    load_tile_rows<kFinRows, 8>(acc, src, nc, f, t0, te, a.x, a.N, f, w, nw);   // x + sum of the partials
#pragma unroll
    for (int k = 0; k < kFinRows; ++k) {
      const int t = t0 + nw * k + w;
      if (t >= te) break;
      const float4 xv = acc[k];
      *reinterpret_cast<float4*>(a.x + (size_t)t * a.N + f) = xv;
      store_act4(a.y_out, (size_t)t * a.N + f, (size_t)kMaxT * a.N,
                 make_float4(g.x * xv.x, g.y * xv.y, g.z * xv.z, g.w * xv.w));
      const float sq = warp_sum(xv.x * xv.x + xv.y * xv.y + xv.z * xv.z + xv.w * xv.w);
      if (l == 0) a.ss_out[(size_t)tile * kMaxT + t] = sq;
    }
  }
}

// EPI_SILU on work tile wt (subtile 0 = gate rows of block wt, subtile 1 = up
// rows), tokens [tb, te), by warp w of nw
template <typename Src>
OOS_DEV void finish_silu(const GemmArgs& a, const Src& src, int wt, int nc, const float* rms, int tb, int te, int w,
                         int nw) {
  const int l = threadIdx.x & 31;
  const int i = wt * kTile + 4 * l;
  constexpr int R = 8;   // 8 token rows per warp per pass
  for (int t0 = tb; t0 < te; t0 += nw * R) {
    float4 gv[R], uv[R];
    // gate and up slices of a pass in one batch of loads
    load_pair_rows<R>(gv, uv, src, nc, 2 * wt * kTile + 4 * l, kTile, t0, te, w, nw);
#pragma unroll
    for (int k = 0; k < R; ++k) {
      const int t = t0 + nw * k + w;
      if (t >= te) break;
      const float r = rms[t];
      const float g4[4] = {gv[k].x * r, gv[k].y * r, gv[k].z * r, gv[k].w * r};
      const float u4[4] = {uv[k].x * r, uv[k].y * r, uv[k].z * r, uv[k].w * r};
      float o4[4];
#pragma unroll
      for (int c = 0; c < 4; ++c) o4[c] = g4[c] / (1.f + expf(-g4[c])) * u4[c];
      store_act4(a.act_out, (size_t)t * a.I + i, (size_t)kMaxT * a.I, make_float4(o4[0], o4[1], o4[2], o4[3]));
    }
  }
}

// EPI_QKV on 128-row tile `tile` = one head (q heads, then k heads, then v
// heads), tokens [tb, te), by warp w of nw
template <typename Src>
OOS_DEV void finish_qkv(const GemmArgs& a, const Src& src, int tile, int nc, const float* rms, int tb, int te, int w,
                        int nw) {
  const int l = threadIdx.x & 31;
  int kind, h;
  if (tile < a.nq) { kind = 0; h = tile; }
  else if (tile < a.nq + a.nkv) { kind = 1; h = tile - a.nq; }
  else { kind = 2; h = tile - a.nq - a.nkv; }
  const __nv_bfloat16* bias = kind == 0 ? a.bq : kind == 1 ? a.bk : a.bv;
  const __nv_bfloat16* gn = kind == 0 ? a.gq : kind == 1 ? a.gk : nullptr;
  const float4 b4 = bias ? bf16x4(bias + h * kTile + 4 * l) : make_float4(0.f, 0.f, 0.f, 0.f);
  const float4 g4 = gn ? bf16x4(gn + 4 * l) : make_float4(1.f, 1.f, 1.f, 1.f);
  const int ctx = *a.ctx;
  const int m0 = 4 * (l & 15);      // rotary frequency index of this lane's first feature
  const bool first_half = l < 16;   // features 0..63 pair with 64..127 held by lane ^ 16
  for (int t0 = tb; t0 < te; t0 += nw * kFinRows) {
    // the pass's rotary factors, loaded ahead of (and so together with) the partial sums
    float2 cs[kFinRows][4];
#pragma unroll
    for (int k = 0; k < kFinRows; ++k) {
      const int t = t0 + nw * k + w;
#pragma unroll
      for (int c = 0; c < 4; ++c)
        cs[k][c] = (kind < 2 && t < te) ? __ldcg(a.rope + t * (kTile / 2) + m0 + c) : make_float2(1.f, 0.f);
    }
    float4 acc[kFinRows];
    load_tile_rows<kFinRows, 8>(acc, src, nc, tile * kTile + 4 * l, t0, te, nullptr, 0, 0, w, nw);
#pragma unroll
    for (int k = 0; k < kFinRows; ++k) {
      const int t = t0 + nw * k + w;
      if (t >= te) break;
      const float r = rms[t];
      float v[4] = {acc[k].x * r + b4.x, acc[k].y * r + b4.y, acc[k].z * r + b4.z, acc[k].w * r + b4.w};
      if (gn) {   // per-head RMSNorm over the head's 128 features
        const float ss = warp_sum(v[0] * v[0] + v[1] * v[1] + v[2] * v[2] + v[3] * v[3]);
        const float rn = rsqrtf(ss * (1.f / kTile) + a.eps);
        v[0] *= rn * g4.x;
        v[1] *= rn * g4.y;
        v[2] *= rn * g4.z;
        v[3] *= rn * g4.w;
      }
      if (kind < 2) {   // rotate-half RoPE at position ctx + depth(t)
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          const float other = __shfl_xor_sync(0xffffffffu, v[c], 16);
          v[c] = first_half ? v[c] * cs[k][c].x - other * cs[k][c].y : v[c] * cs[k][c].x + other * cs[k][c].y;
        }
      }
      if (kind == 0) {   // q as hi/lo halves in the cache's 16-bit format: the attention product sees ~16-bit q
        const size_t qi = ((size_t)t * a.nq + h) * kTile + 4 * l, lo_off = (size_t)kMaxT * a.nq * kTile;
        if (a.kv_f16) store_act4_h(reinterpret_cast<__half*>(a.q_out), qi, lo_off, make_float4(v[0], v[1], v[2], v[3]));
        else store_act4(a.q_out, qi, lo_off, make_float4(v[0], v[1], v[2], v[3]));
      } else {           // K/V in the cache's format (bf16, or binary16)
        __nv_bfloat16* dst = (kind == 1 ? a.kc : a.vc) + ((size_t)(ctx + t) * a.nkv + h) * kTile;
        uint2 o;
        if (a.kv_f16) {
          __half hv[4];
#pragma unroll
          for (int c = 0; c < 4; ++c) hv[c] = __float2half_rn(v[c]);
          o = *reinterpret_cast<const uint2*>(hv);
        } else {
          __nv_bfloat16 bv[4];
#pragma unroll
          for (int c = 0; c < 4; ++c) bv[c] = __float2bfloat16_rn(v[c]);
          o = *reinterpret_cast<const uint2*>(bv);
        }
        *reinterpret_cast<uint2*>(dst + 4 * l) = o;
      }
    }
  }
}

template <int BN, int EPI>
__global__ void __launch_bounds__(192, 1)
    k_gemm_tc(const __grid_constant__ CUtensorMap wm0, const __grid_constant__ CUtensorMap wm1,
              const __grid_constant__ CUtensorMap wm2, const __grid_constant__ CUtensorMap am, GemmArgs a) {
  constexpr int kSub = SubOf<EPI>::v;
  using C = TcCfg<BN, kSub>;
  constexpr int S = C::S;
  constexpr bool ARGMAX = EPI == EPI_ARGMAX;
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  // stage layout: [A subtile 0 | A subtile 1 | B hi | B lo]
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S * C::STAGE);
  uint64_t* empty = full + S;
  uint64_t* accf = empty + S;
  uint64_t* acce = accf + 2;
  uint64_t* drain = acce + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  float* rms = reinterpret_cast<float*>(smem + S * C::STAGE + C::BAR_BYTES);       // [kMaxT]
  Top2s* red = reinterpret_cast<Top2s*>(smem + S * C::STAGE + C::BAR_BYTES + C::EPI_BYTES);   // [4][BN]
  Top2s* run = red + 4 * BN;                                                                   // [BN]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = gridDim.x, cta = blockIdx.x;
  if (threadIdx.x == 0) TL_GEMM(0);

  // this CTA's work: units [u0, u1) (stream-K) or work tiles cta, cta+G, ... (LM head)
  long long u0, u1;
  if (!ARGMAX) {
    u0 = (long long)cta * a.total / G;
    u1 = (long long)(cta + 1) * a.total / G;
  } else {
    const int my_tiles = cta < a.n_work ? (a.n_work - cta + G - 1) / G : 0;
    u0 = 0;
    u1 = (long long)my_tiles * a.kbt;
  }
  const int n_units = (int)(u1 - u0);
  auto unit_tile = [&](int j, int& wt, int& kb) {
    if (!ARGMAX) {
      const long long u = u0 + j;
      wt = (int)(u / a.kbt);
      kb = (int)(u % a.kbt);
    } else {
      wt = cta + (j / a.kbt) * G;
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
    abort_flag[0] = 0;
    abort_flag[1] = 0;
    mbar_fence_init();
  }
  if (warp == 2) tmem_alloc(tmem_slot, C::NCOLS);
  if (ARGMAX && threadIdx.x >= 64) {
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
        int wt, kb;
        unit_tile(j, wt, kb);
#pragma unroll
        for (int sub = 0; sub < kSub; ++sub) {
          const int tile = wt * kSub + sub;          // 128-row tile of the stacked weight
          const CUtensorMap* wm = &wm0;
          int row = tile * kTile;
          if (a.interleave2) {
            wm = (tile & 1) ? &wm1 : &wm0;
            row = (tile >> 1) * kTile;
          } else if (tile >= a.seg_tiles[0]) {
            if (tile >= a.seg_tiles[1]) {
              wm = &wm2;
              row = (tile - a.seg_tiles[1]) * kTile;
            } else {
              wm = &wm1;
              row = (tile - a.seg_tiles[0]) * kTile;
            }
          }
          // a subtile past the last weight row reads zeros (TMA out-of-bounds fill)
          tma_load_2d(smem + stage * C::STAGE + sub * C::A_BYTES, wm, &full[stage], kb * kBK, row, pol_w);
        }
      };
      auto load_x = [&](int j, int stage) {
        int wt, kb;
        unit_tile(j, wt, kb);
        unsigned char* dst = smem + stage * C::STAGE + kSub * C::A_BYTES;
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
      pdl_trigger();
      TL_GEMM(1);
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
      {
        // every copy this thread issued has landed before the CTA can exit,
        // whoever gave up (immediate on the normal path, where all were consumed)
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
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(kTile, C::PAIRED ? 2 * BN : BN);
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_use[2] = {0, 0};
      int j = 0;
      bool ok = true;
      while (j < n_units && ok) {
        int wt, kb;
        unit_tile(j, wt, kb);
        int seg_end = j + (a.kbt - kb);       // units of this work tile owned here
        if (seg_end > n_units) seg_end = n_units;
        if (!mbar_wait(&acce[acc], (acc_use[acc] & 1u) ^ 1u, abort_flag, a.status)) break;
        tc_fence_after();
        const uint32_t d0 = tmem_base + (uint32_t)(acc * kSub * C::SUB_COLS);
        for (int jj = j; jj < seg_end; ++jj) {
          if (!mbar_wait(&full[stage], phase, abort_flag, a.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sbase = smem_addr(smem + stage * C::STAGE);
          const uint64_t bh = smem_desc_sw128(sbase + kSub * C::A_BYTES);
          const uint64_t bl = smem_desc_sw128(sbase + kSub * C::A_BYTES + C::B_BYTES);
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k) {
#pragma unroll
            for (int sub = 0; sub < kSub; ++sub) {
              const uint64_t ad = smem_desc_sw128(sbase + sub * C::A_BYTES);
              const uint32_t d = d0 + (uint32_t)(sub * C::SUB_COLS);
              tc_mma_bf16(d, ad + 2 * k, bh + 2 * k, idesc, (jj > j || k > 0) ? 1u : 0u);
              if (!C::PAIRED) tc_mma_bf16(d, ad + 2 * k, bl + 2 * k, idesc, 1u);
            }
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
    pdl_trigger();
    const int q = warp & 3;               // TMEM lane quarter this warp may access
    const int row = q * 32 + lane;
    const int e = threadIdx.x - 64;       // 0..127
    // Abort decisions of the epilogue warps are taken on one sample of the
    // flag, so all 128 threads leave together and no named barrier is left
    // waiting for threads that have gone.
    volatile int* epi_abort = abort_flag + 1;
    auto epi_aborted = [&]() -> bool {
      epi_bar();
      if (e == 0) *epi_abort = *abort_flag;
      epi_bar();
      return *epi_abort != 0;
    };
    if (EPI != EPI_RESID) {
      if (e < a.T) {
        float s = 0.f;
        for (int c = 0; c < a.ss_chunks; ++c) s += a.ss_in[(size_t)c * kMaxT + e];
        rms[e] = rsqrtf(s * a.inv_dim + a.eps);
      }
      epi_bar();
    }
    const int n_part = a.n_work * kSub * kTile;
    int acc = 0;
    uint32_t acc_use[2] = {0, 0};
    int j = 0;
    while (j < n_units) {
      int wt, kb;
      unit_tile(j, wt, kb);
      int seg_end = j + (a.kbt - kb);
      if (seg_end > n_units) seg_end = n_units;
      mbar_wait(&accf[acc], acc_use[acc] & 1u, abort_flag, a.status);
      if (e == 0 && seg_end >= n_units) TL_GEMM(2);
      if (epi_aborted()) break;
      tc_fence_after();
      const uint32_t taddr0 = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * kSub * C::SUB_COLS);
      // 16 accumulator columns (tokens) of subtile `sub`: paired hi + lo products
      auto acc16 = [&](int sub, int cc, float (&v)[16]) {
        tmem_ld16(taddr0 + sub * C::SUB_COLS + cc * 16, v);
        if (C::PAIRED) {
          float w[16];
          tmem_ld16(taddr0 + sub * C::SUB_COLS + BN + cc * 16, w);
#pragma unroll
          for (int i = 0; i < 16; ++i) v[i] += w[i];
        }
      };
      if (!ARGMAX) {
        int c0, c1;
        StreamK sk{a.n_work, a.kbt, a.total, G};
        sk.contributors(wt, c0, c1);
        // lane l holds row q*32 + l; a 4 x 4 shuffle transpose per 4 tokens gives
        // each lane 4 consecutive rows of one token: one float4 store, not four
        const int li = lane & 3;
#pragma unroll 1
        for (int sub = 0; sub < kSub; ++sub) {
          float* dst = a.part + (size_t)(cta - c0) * kMaxT * n_part + (size_t)(wt * kSub + sub) * kTile + q * 32 +
                       (lane & ~3);
          // the subtile's accumulator row in batches of TMEM loads (up to 64
          // tokens, hi and lo products when paired), one wait per batch
          constexpr int NG = BN / 16 < 4 ? BN / 16 : 4;   // 16-token chunks per batch
#pragma unroll 1
          for (int c0g = 0; c0g < BN / 16; c0g += NG) {
            if (c0g * 16 >= a.T) break;
            float vv[NG][16], ww[C::PAIRED ? NG : 1][16];
#pragma unroll
            for (int k = 0; k < NG; ++k) {
              tmem_ld16_nowait(taddr0 + sub * C::SUB_COLS + (c0g + k) * 16, vv[k]);
              if (C::PAIRED) tmem_ld16_nowait(taddr0 + sub * C::SUB_COLS + BN + (c0g + k) * 16, ww[C::PAIRED ? k : 0]);
            }
            tmem_wait_ld();
#pragma unroll
            for (int k = 0; k < NG; ++k) {
              reg_fence(vv[k]);
              if (C::PAIRED) reg_fence(ww[C::PAIRED ? k : 0]);
            }
#pragma unroll
          for (int k = 0; k < NG; ++k) {
            const int cc = c0g + k;
            if (cc * 16 >= a.T) break;
            float v[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) v[i] = C::PAIRED ? vv[k][i] + ww[C::PAIRED ? k : 0][i] : vv[k][i];
#pragma unroll
            for (int b = 0; b < 4; ++b) {
              float x0 = v[4 * b], x1 = v[4 * b + 1], x2 = v[4 * b + 2], x3 = v[4 * b + 3];
              const float y0 = __shfl_xor_sync(0xffffffffu, (li & 1) ? x0 : x1, 1);
              const float y1 = __shfl_xor_sync(0xffffffffu, (li & 1) ? x2 : x3, 1);
              if (li & 1) {
                x0 = y0;
                x2 = y1;
              } else {
                x1 = y0;
                x3 = y1;
              }
              const float z0 = __shfl_xor_sync(0xffffffffu, (li & 2) ? x0 : x2, 2);
              const float z1 = __shfl_xor_sync(0xffffffffu, (li & 2) ? x1 : x3, 2);
              if (li & 2) {
                x0 = z0;
                x1 = z1;
              } else {
                x2 = z0;
                x3 = z1;
              }
              const int t = cc * 16 + 4 * b + li;   // rows (lane & ~3) .. +3 of token t
              if (t < a.T) *reinterpret_cast<float4*>(dst + (size_t)t * n_part) = make_float4(x0, x1, x2, x3);
            }
          }
          }
        }
        // accumulators drained: hand the TMEM buffer back to the MMA issuer
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&acce[acc]);
        // publish this contribution (finished at the end of the range)
        __threadfence();
        epi_bar();
        if (e == 0) atomicAdd(&a.cnt[wt], 1);
        if (e == 0 && seg_end >= n_units) TL_GEMM(4);
      } else {
#pragma unroll 1
        for (int sub = 0; sub < kSub; ++sub) {
          const int f = (wt * kSub + sub) * kTile + row;
#pragma unroll 1
          for (int cc = 0; cc < BN / 16; ++cc) {
            if (cc * 16 >= a.T) break;
            float v[16];
            acc16(sub, cc, v);
#pragma unroll
            for (int i = 0; i < 16; ++i) {
              Top2s s{f < a.N ? v[i] * rms[cc * 16 + i] : -INFINITY, f, -INFINITY};
#pragma unroll
              for (int o = 16; o > 0; o >>= 1) {
                Top2s y;
                y.v1 = __shfl_xor_sync(0xffffffffu, s.v1, o);
                y.i1 = __shfl_xor_sync(0xffffffffu, s.i1, o);
                y.v2 = __shfl_xor_sync(0xffffffffu, s.v2, o);
                s = t2_merge(s, y);
              }
              if (lane == 0) {
                Top2s* slot = &red[q * BN + cc * 16 + i];
                *slot = sub == 0 ? s : t2_merge(*slot, s);
              }
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&acce[acc]);
        epi_bar();
        if (e < a.T) {
          Top2s r = run[e];
#pragma unroll
          for (int w = 0; w < 4; ++w) r = t2_merge(r, red[w * BN + e]);
          run[e] = r;
        }
        epi_bar();
      }
      ++acc_use[acc];
      acc ^= 1;
      j = seg_end;
    }
    if (!ARGMAX && !epi_aborted()) {
      // Finish every work tile this CTA touched: once all nc contributions of
      // the tile have arrived, contributor i (in CTA order) finishes token rows
      // [T*i/nc, T*(i+1)/nc) -- slices are still added in slice order, so the
      // result does not depend on who finishes.  All contributors end their
      // ranges at about the same time (balanced stream-K), and the grid never
      // exceeds one CTA per SM, so every awaited CTA is resident.  Tiles are
      // taken two at a time: both arrival counts are awaited first, then
      // epilogue warps 0-1 finish the first tile and warps 2-3 the second, so
      // the two latency-bound passes overlap instead of running back to back.
      StreamK sk{a.n_work, a.kbt, a.total, G};
      int jj = 0;
      bool tl_first = true;
      while (jj < n_units) {
        // the next one or two work tiles of the range: (tile, contributors, token share)
        auto next_tile = [&](int& wt, int& nc, int& tb, int& te) {
          int kb;
          unit_tile(jj, wt, kb);
          int seg_end = jj + (a.kbt - kb);
          if (seg_end > n_units) seg_end = n_units;
          jj = seg_end;
          int c0, c1;
          sk.contributors(wt, c0, c1);
          nc = c1 - c0 + 1;
          const int share = cta - c0;
          tb = (int)((long long)a.T * share / nc);
          te = (int)((long long)a.T * (share + 1) / nc);
        };
        int wt0, nc0, tb0, te0, wt1 = -1, nc1 = 0, tb1 = 0, te1 = 0;
        next_tile(wt0, nc0, tb0, te0);
        if (jj < n_units) next_tile(wt1, nc1, tb1, te1);
        const bool two = wt1 >= 0;
        if (e == 0) {
          const unsigned long long t0 = globaltimer();
          const unsigned long long limit = wait_limit(a.status);
          for (int i = 0; i < (two ? 2 : 1) && !*abort_flag; ++i) {
            const int wt = i ? wt1 : wt0, nc = i ? nc1 : nc0;
            while (*(volatile int*)&a.cnt[wt] < nc) {
              if (*abort_flag || (*(volatile uint32_t*)a.status & ST_TIMEOUT)) {
                *abort_flag = 1;
                break;
              }
              if (globaltimer() - t0 > limit) {
                atomicOr(a.status, ST_TIMEOUT);
                *abort_flag = 1;
                break;
              }
            }
          }
        }
        if (epi_aborted()) break;
        if (e == 0 && tl_first) TL_GEMM(5);
        tl_first = false;
        __threadfence();
        const int ew = e >> 5;   // epilogue warp 0..3
        const bool second = two && ew >= 2;
        const int nw = two ? 2 : 4, w = two ? (ew & 1) : ew;
        const int wt = second ? wt1 : wt0, nc = second ? nc1 : nc0, tb = second ? tb1 : tb0, te = second ? te1 : te0;
        if (tb < te) {
          const GSrc src{a.part, (size_t)kMaxT * n_part, n_part};
          if (EPI == EPI_SILU) {
            finish_silu(a, src, wt, nc, rms, tb, te, w, nw);
          } else {
#pragma unroll 1
            for (int sub = 0; sub < kSub; ++sub) {
              const int tile = wt * kSub + sub;
              if (tile >= a.n_tiles) break;
              if (EPI == EPI_RESID) finish_resid(a, src, tile, nc, tb, te, w, nw);
              else finish_qkv(a, src, tile, nc, rms, tb, te, w, nw);
            }
          }
        }
      }
    }
    if (ARGMAX && e < a.T) {
      const Top2s r = run[e];
      a.am_v1[(size_t)cta * kMaxT + e] = r.v1;
      a.am_i[(size_t)cta * kMaxT + e] = r.i1;
      a.am_v2[(size_t)cta * kMaxT + e] = r.v2;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0) TL_GEMM(3);
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

bool encode_bf16_map(CUtensorMap* map, const void* ptr, int rank, const uint64_t* dims, const uint64_t* strides,
                     const uint32_t* box, bool f16) {
  EncodeTiledFn enc = get_encode();
  if (!enc || rank < 1 || rank > 5) return false;
  memset(map, 0, sizeof(*map));
  cuuint64_t gdim[5], gstride[4];
  cuuint32_t bx[5], estr[5];
  for (int i = 0; i < rank; ++i) {
    gdim[i] = dims[i];
    bx[i] = box[i];
    estr[i] = 1;
    if (i + 1 < rank) gstride[i] = strides[i];
  }
  CUresult r = enc(map, f16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, (cuuint32_t)rank,
                   const_cast<void*>(ptr), gdim, gstride, bx,
                   estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
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

template <int BN, int EPI>
static cudaError_t set_smem() {
  cudaError_t e = cudaFuncSetAttribute(k_gemm_tc<BN, EPI>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       TcCfg<BN, SubOf<EPI>::v>::SMEM);
  return e;
}


template <int BN>
static cudaError_t set_smem_all() {
  cudaError_t e = set_smem<BN, EPI_QKV>();
  if (e == cudaSuccess) e = set_smem<BN, EPI_RESID>();
  if (e == cudaSuccess) e = set_smem<BN, EPI_SILU>();
  if (e == cudaSuccess) e = set_smem<BN, EPI_ARGMAX>();
  return e;
}

cudaError_t gemm_setup() {
  cudaError_t e = set_smem_all<16>();
  if (e == cudaSuccess) e = set_smem_all<32>();
  if (e == cudaSuccess) e = set_smem_all<64>();
  if (e == cudaSuccess) e = set_smem_all<128>();
  return e;
}

template <int BN, int EPI>
static cudaError_t launch_tc(Model& m, const GemmW& g, const CUtensorMap& amap, int grid, const GemmArgs& a,
                             cudaStream_t st) {
  const CUtensorMap& w1 = g.n_seg > 1 ? g.map[1] : g.map[0];
  const CUtensorMap& w2 = g.n_seg > 2 ? g.map[2] : g.map[0];
  return launch(m.pdl, k_gemm_tc<BN, EPI>, dim3(grid), dim3(192), (size_t)TcCfg<BN, SubOf<EPI>::v>::SMEM, st,
                g.map[0], w1, w2, amap, a);
}

template <int EPI>
static cudaError_t dispatch_tc(Model& m, const GemmW& g, const CUtensorMap* amaps, int T, int grid, GemmArgs& a,
                               cudaStream_t st) {
  const int bi = bn_index(T);
  switch (bi) {
    case 0: return launch_tc<16, EPI>(m, g, amaps[0], grid, a, st);
    case 1: return launch_tc<32, EPI>(m, g, amaps[1], grid, a, st);
    case 2: return launch_tc<64, EPI>(m, g, amaps[2], grid, a, st);
    default: return launch_tc<128, EPI>(m, g, amaps[3], grid, a, st);
  }
}

int* gemm_counters(Model& m, int layer, int kind) { return m.ws.cnt + ((size_t)layer * 4 + kind) * kCntPer; }

static GemmArgs base_args(Model& m, const GemmW& g, int T, int* cnt) {
  GemmArgs a;
  memset(&a, 0, sizeof(a));
  for (int s = 0; s < 3; ++s) a.seg_tiles[s] = g.seg_tiles[s < g.n_seg ? s : g.n_seg - 1];
  a.interleave2 = g.interleave2;
  a.n_tiles = (g.N + kTile - 1) / kTile;
  a.n_work = g.plan.n_tiles;
  a.kbt = g.plan.kbt;
  a.total = g.plan.total;
  a.N = g.N;
  a.T = T;
  a.part = m.ws.part;
  a.cnt = cnt;
  a.status = m.ws.status;
  a.ss_in = m.ws.ss;
  a.ss_chunks = (m.cfg.hidden + kTile - 1) / kTile;
  a.inv_dim = 1.0f / (float)m.cfg.hidden;
  a.eps = m.cfg.rms_eps;
  return a;
}

cudaError_t launch_gemm_qkv(Model& m, int layer, void* kc, void* vc, int T, cudaStream_t st) {
  const auto& c = m.cfg;
  const oos_layer_weights& L = m.layers[layer];
  GemmArgs a = base_args(m, m.g_qkv[layer], T, gemm_counters(m, layer, 0));
  a.nq = c.n_q_heads;
  a.nkv = c.n_kv_heads;
  a.bq = (const __nv_bfloat16*)(c.qkv_bias ? L.b_q : nullptr);
  a.bk = (const __nv_bfloat16*)(c.qkv_bias ? L.b_k : nullptr);
  a.bv = (const __nv_bfloat16*)(c.qkv_bias ? L.b_v : nullptr);
  a.gq = (const __nv_bfloat16*)(c.qk_norm ? L.q_norm : nullptr);
  a.gk = (const __nv_bfloat16*)(c.qk_norm ? L.k_norm : nullptr);
  a.rope = m.ws.rope;
  a.q_out = (__nv_bfloat16*)m.ws.q;
  a.kc = (__nv_bfloat16*)kc;
  a.vc = (__nv_bfloat16*)vc;
  a.ctx = m.ws.ctx;
  a.kv_f16 = c.kv_f16 ? 1 : 0;
  return dispatch_tc<EPI_QKV>(m, m.g_qkv[layer], m.amap_xn, T, m.g_qkv[layer].plan.grid, a, st);
}

static cudaError_t launch_resid(Model& m, const GemmW& g, const CUtensorMap* amaps, const void* gain, int* cnt, int T,
                                cudaStream_t st) {
  GemmArgs a = base_args(m, g, T, cnt);
  a.x = m.ws.x;
  a.gain = (const __nv_bfloat16*)gain;
  a.y_out = (__nv_bfloat16*)m.ws.xn;
  a.ss_out = m.ws.ss;
  return dispatch_tc<EPI_RESID>(m, g, amaps, T, g.plan.grid, a, st);
}

cudaError_t launch_gemm_o(Model& m, int layer, int T, cudaStream_t st) {
  return launch_resid(m, m.g_o[layer], m.amap_attn, m.layers[layer].mlp_norm, gemm_counters(m, layer, 1), T, st);
}

cudaError_t launch_gemm_down(Model& m, int layer, int T, cudaStream_t st) {
  const void* gain = layer + 1 < m.cfg.n_layers ? m.layers[layer + 1].attn_norm : m.w.final_norm;
  return launch_resid(m, m.g_down[layer], m.amap_act, gain, gemm_counters(m, layer, 3), T, st);
}

cudaError_t launch_gemm_gu(Model& m, int layer, int T, cudaStream_t st) {
  GemmArgs a = base_args(m, m.g_gu[layer], T, gemm_counters(m, layer, 2));
  a.act_out = (__nv_bfloat16*)m.ws.act;
  a.I = m.cfg.intermediate;
  return dispatch_tc<EPI_SILU>(m, m.g_gu[layer], m.amap_xn, T, m.g_gu[layer].plan.grid, a, st);
}

cudaError_t launch_lm_head_tc(Model& m, int T, cudaStream_t st) {
  GemmArgs a = base_args(m, m.g_lm, T, nullptr);
  a.am_v1 = m.ws.lm_v1;
  a.am_i = m.ws.lm_i;
  a.am_v2 = m.ws.lm_v2;
  return dispatch_tc<EPI_ARGMAX>(m, m.g_lm, m.amap_xn, T, m.lm_grid, a, st);
}

// ------------------------------------------------------------ fp32 CUDA-core path
// One warp per output row; part[t][f] = W[f] . x[t] (a single slice).
__global__ void __launch_bounds__(128) k_gemm_f32(const float* __restrict__ w0, const float* __restrict__ w1,
                                                  const float* __restrict__ w2, int r0, int r1, int r2, int K,
                                                  const float* __restrict__ x, int T, float* __restrict__ part) {
  pdl_wait();
  pdl_trigger();
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
  pdl_trigger();
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
}

cudaError_t launch_lm_head_f32(Model& m, int T, cudaStream_t st) {
  const int V = m.cfg.vocab;
  const int rows = (V + m.lm_grid - 1) / m.lm_grid;
  return launch(m.pdl, k_lm_head_f32, dim3(m.lm_grid), dim3(128), 0, st, (const float*)m.w.lm_head, V, m.cfg.hidden,
                rows, (const float*)m.ws.xn, T, m.ws.lm_v1, m.ws.lm_i, m.ws.lm_v2);
}

}  // namespace oos

#ifdef OOS_TIMELINE
// timeline accessors (the OOS_TIMELINE library only)
extern "C" int oos_timeline_gemm_read(void* out, size_t bytes) {
  return cudaMemcpyFromSymbol(out, oos::g_tl_gemm, bytes < sizeof(oos::g_tl_gemm) ? bytes : sizeof(oos::g_tl_gemm)) ==
                 cudaSuccess
             ? 0
             : OOS_ECUDA;
}
extern "C" int oos_timeline_gemm_clear() {
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, oos::g_tl_gemm) != cudaSuccess) return OOS_ECUDA;
  return cudaMemset(p, 0, sizeof(oos::g_tl_gemm)) == cudaSuccess ? 0 : OOS_ECUDA;
}
#endif
