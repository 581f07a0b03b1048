// bf16 projections of the depth-sparse layer on the 5th-generation tensor cores.
//
// out = epilogue(A . W^T) with A [M, K] (packed kept tokens, row-major) and
// W [N, K] (nn.Linear layout); both operands are K-major, which is the layout
// tcgen05 reads natively. These are the dense contractions of Eqs. 1-2 (QKV,
// output and MLP projections) and the router's first linear layer (Sec. 3.4).
//
// Kernel structure (one persistent CTA per SM, 10 warps):
//   warp 0     TMA producer: 128x64 A tile and BNx64 W tile(s) per stage into a
//              STAGES-deep shared-memory ring, 128-byte swizzled, signalled
//              through mbarrier transaction counts.
//   warp 1     allocates TMEM; one thread issues tcgen05.mma (M=128, N=BN,
//              K=16, fp32 accumulator in TMEM) and commits stage releases and
//              accumulator hand-offs to mbarriers.
//   warps 2-9  epilogue: tcgen05.ld the accumulator (one row per thread, two
//              warps per 32-lane TMEM quarter splitting the columns), apply
//              bias / GELU / SwiGLU / rotary / residual / row scatter / router
//              reduction in fp32, round once and store.
// The accumulator is double-buffered in TMEM so the epilogue of tile i runs
// under the main loop of tile i+1. Every barrier wait is bounded in time; on
// give-up the CTA records DEVERR_TIMEOUT, drains its in-flight copies and
// MMAs, frees TMEM and exits.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>

#include "common.cuh"
#include "internal.h"

namespace adadsf {
namespace {

constexpr int BM = 128;
constexpr int BK = 64;       // one 128-byte swizzle row of bf16
constexpr int UK = 16;       // K of one tcgen05.mma kind::f16
constexpr int kEpiWarps = 8;     // two per TMEM lane quarter, each on half of the columns
constexpr int kThreads = 64 + 32 * kEpiWarps;
constexpr int kGroupM = 16;  // tile raster: 16 M-blocks share each W column block

// PAIR: two-CTA variant. Plain: each CTA stages half of the BN weight rows.
// DUAL: the even CTA stages BN rows of the first weight, the odd CTA BN rows
// of the second, so one N = 2 BN pair MMA yields both accumulators.
template <int BN, bool DUAL, bool PAIR = false>
struct TileCfg {
  static constexpr int A_BYTES = BM * BK * 2;
  static constexpr int B_ROWS = (PAIR && !DUAL) ? BN / 2 : BN;
  static constexpr int B_BYTES = B_ROWS * BK * 2;
  static constexpr int NUM_B = (DUAL && !PAIR) ? 2 : 1;   // weight tiles per stage
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES * NUM_B;
  static constexpr int STAGES_FIT = 196608 / STAGE_BYTES;
  static constexpr int STAGES = STAGES_FIT > 8 ? 8 : STAGES_FIT;
  static constexpr int ACC_COLS = BN * (DUAL ? 2 : 1);
  static constexpr int TMEM_COLS = 2 * ACC_COLS;
  static constexpr int BAR_BYTES = (2 * STAGES + 5) * 8 + 16;
  static constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + 1024 + BAR_BYTES;
  static_assert(TMEM_COLS == 128 || TMEM_COLS == 256 || TMEM_COLS == 512, "TMEM columns");
  static_assert(SMEM_BYTES <= 232448, "shared memory");
};

struct GemmDev {
  int M, N, K;
  int act;
  const bf16* bias;
  const bf16* add_packed; int64_t ld_add_packed;
  const bf16* add_rows;   int64_t ld_add_rows;
  const int32_t* rows;
  int out_mapped;
  bf16* out; int64_t ld_out;
  const bf16* w2; const bf16* b2; float* scores;
  // rotary embedding fused into the QKV epilogue (rope_tab == nullptr: off)
  const float2* rope_tab;    // [T][rope_half] (cos, sin)
  const int32_t* rope_pos;   // [M] original positions, or null: m % rope_T
  int rope_T, rope_half, rope_hd, rope_cols;
  bf16* vt;                  // transposed value heads (see Epilogue::vt)
  int vt_seq, vt_pad, vt_col0, vt_hd, vt_hkv;
  int* err;
  unsigned long long timeout_ns;
};

__device__ __forceinline__ void tile_coords(int t, int num_m, int num_n, int& mb, int& nb) {
  const int group_tiles = kGroupM * num_n;
  const int g = t / group_tiles;
  const int first_m = g * kGroupM;
  const int gsz = min(num_m - first_m, kGroupM);
  const int r = t - g * group_tiles;
  mb = first_m + r % gsz;
  nb = r / gsz;
}

__device__ __forceinline__ float gelu_f(float v) { return 0.5f * v * (1.f + erff(v * 0.70710678118654752f)); }
__device__ __forceinline__ float silu_f(float v) { return v / (1.f + expf(-v)); }

// Epilogue of one 32-column chunk of one row (all values fp32 in v[]).
__device__ __forceinline__ void epi_chunk_store(const GemmDev& p, float* v, int m, int64_t arow,
                                                int64_t orow, int n0) {
  if (p.add_packed) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      float f[8];
      load_vec(p.add_packed + (int64_t)m * p.ld_add_packed + n0 + 8 * i, f);
#pragma unroll
      for (int j = 0; j < 8; ++j) v[8 * i + j] += f[j];
    }
  }
  if (p.add_rows) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      float f[8];
      load_vec(p.add_rows + arow * p.ld_add_rows + n0 + 8 * i, f);
#pragma unroll
      for (int j = 0; j < 8; ++j) v[8 * i + j] += f[j];
    }
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) store_vec(p.out + orow * p.ld_out + n0 + 8 * i, v + 8 * i);
}

// Rotates the pairs (a[j], b[j]) j < n by the angles of features i0 + j at
// the row's position: a' = a cos - b sin, b' = b cos + a sin.
__device__ __forceinline__ void rope_rotate(float* a, float* b, int n, const float2* tab_row, int i0) {
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    if (j < n) {
      const float2 cs = tab_row[i0 + j];
      const float x = a[j], y = b[j];
      a[j] = x * cs.x - y * cs.y;
      b[j] = y * cs.x + x * cs.y;
    }
  }
}

// Feature j < H of the chunk pairs with feature j + H (H = rotary half <= 16).
template <int H>
__device__ __forceinline__ void rope_in_chunk(float* v, const float2* tab_row) {
#pragma unroll
  for (int j = 0; j < H; ++j) {
    const float2 cs = tab_row[j];
    const float x = v[j], y = v[j + H];
    v[j] = x * cs.x - y * cs.y;
    v[j + H] = y * cs.x + x * cs.y;
  }
}

__device__ __forceinline__ void add_bias32(const bf16* bias, int n0, float* v) {
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    float f[8];
    load_vec(bias + n0 + 8 * i, f);
#pragma unroll
    for (int j = 0; j < 8; ++j) v[8 * i + j] += f[j];
  }
}

// Epilogue of one accumulator tile for the calling thread's row m: chunks of
// 32 TMEM columns (this warp's half of them) -> bias / activation / rotary /
// residual / store, or the router's row reduction.
template <int BN, bool DUAL, bool ROUTER>
__device__ __forceinline__ void epilogue_tile(const GemmDev& p, uint32_t tacc, int m, int nb,
                                              int half) {
  const bool rope = !ROUTER && !DUAL && p.rope_tab != nullptr;
  const bool mvalid = m < p.M;
  int64_t arow = m;
  if (mvalid && p.rows) arow = p.rows[m];
  const int64_t orow = p.out_mapped ? arow : (int64_t)m;
  const float2* tab_row = nullptr;
  if (rope && mvalid)
    tab_row = p.rope_tab + (int64_t)(p.rope_pos ? p.rope_pos[m] : m % p.rope_T) * p.rope_half;
  float rsum = 0.f;
  constexpr int NC = BN / 32;
#pragma unroll 1
  for (int c = 0; c < NC; ++c) {
    // the router's row reduction stays in one warp per quarter
    const int owner = ROUTER ? 0 : (c < NC / 2 ? 0 : 1);
    if (owner != half) continue;
    const int n0 = nb * BN + c * 32;
    // rotary halves of 32 or more features: chunk c pairs with chunk c2,
    // both handled by the owner of c
    const bool rot = rope && n0 < p.rope_cols;
    const bool paired = rot && p.rope_half >= 32;
    if (paired && (n0 % p.rope_hd) >= p.rope_half) continue;   // done with its partner
    const int c2 = paired ? c + p.rope_half / 32 : c;
    uint32_t r[32];
    uint32_t r2[(DUAL || !ROUTER) ? 32 : 1];
    tmem_ld32(tacc + c * 32, r);
    if (DUAL) tmem_ld32(tacc + BN + c * 32, r2);
    else if (!ROUTER && paired) tmem_ld32(tacc + c2 * 32, r2);
    tmem_ld_wait();
    if (!mvalid || n0 >= p.N) continue;
    float v[32];
#pragma unroll
    for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
    if (p.bias) add_bias32(p.bias, n0, v);
    if (!ROUTER && !DUAL && p.vt && n0 >= p.vt_col0) {
      // value columns: also store this row's 32 features transposed
      const int vc = n0 - p.vt_col0;
      const int bseq = m / p.vt_seq, j = m - bseq * p.vt_seq;
      bf16* dst = p.vt + ((int64_t)(bseq * p.vt_hkv + vc / p.vt_hd) * p.vt_hd + vc % p.vt_hd) *
                             p.vt_pad + j;
#pragma unroll
      for (int i = 0; i < 32; ++i) dst[(int64_t)i * p.vt_pad] = __float2bfloat16_rn(v[i]);
    }
    if (ROUTER) {
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        float f[8];
        load_vec(p.w2 + n0 + 8 * i, f);
#pragma unroll
        for (int j = 0; j < 8; ++j) rsum += f[j] * silu_f(v[8 * i + j]);
      }
      continue;
    }
    if (DUAL) {
#pragma unroll
      for (int j = 0; j < 32; ++j) v[j] = silu_f(v[j]) * __uint_as_float(r2[j]);
    } else if (p.act == ACT_GELU) {
#pragma unroll
      for (int j = 0; j < 32; ++j) v[j] = gelu_f(v[j]);
    }
    if (!DUAL && paired) {
      const int n2 = nb * BN + c2 * 32;
      float v2[32];
#pragma unroll
      for (int j = 0; j < 32; ++j) v2[j] = __uint_as_float(r2[j]);
      if (p.bias) add_bias32(p.bias, n2, v2);
      rope_rotate(v, v2, 32, tab_row, n0 % p.rope_hd);
      epi_chunk_store(p, v2, m, arow, orow, n2);
    } else if (rot && (n0 % p.rope_hd) == 0) {
      // rotary half of at most 16 features: both halves inside this chunk
      switch (p.rope_half) {
        case 4: rope_in_chunk<4>(v, tab_row); break;
        case 8: rope_in_chunk<8>(v, tab_row); break;
        case 16: rope_in_chunk<16>(v, tab_row); break;
        default: break;
      }
    }
    epi_chunk_store(p, v, m, arow, orow, n0);
  }
  if (ROUTER && half == 0 && mvalid) p.scores[m] = rsum + __bfloat162float(p.b2[0]);
}

template <int BN, bool DUAL, bool ROUTER>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ CUtensorMap tmB2, const GemmDev p) {
  using C = TileCfg<BN, DUAL>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const uint32_t sA = smem_u32(smem);
  const uint32_t sB = sA + C::STAGES * C::A_BYTES;
  const uint32_t sB2 = sB + C::STAGES * C::B_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::STAGES * C::STAGE_BYTES);
  const uint32_t full0 = smem_u32(bars);
  const uint32_t empty0 = full0 + 8 * C::STAGES;
  const uint32_t tfull0 = empty0 + 8 * C::STAGES;
  const uint32_t tempty0 = tfull0 + 16;
  const uint32_t drain = tempty0 + 16;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * C::STAGES + 5);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int num_m = (p.M + BM - 1) / BM;
  const int num_n = (p.N + BN - 1) / BN;
  const int num_kb = (p.K + BK - 1) / BK;
  const int num_tiles = num_m * num_n;

  pdl_trigger();
  if (threadIdx.x == 0) {
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(tfull0 + 8 * a, 1);
      mbar_init(tempty0 + 8 * a, kEpiWarps);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_barrier_init();
    fence_proxy_async_smem();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
    if (DUAL) tma_prefetch_desc(&tmB2);
  }
  if (warp == 1) tmem_alloc(smem_u32(tmem_slot), C::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int64_t issued = 0;
      constexpr uint32_t tx = C::STAGE_BYTES;
      // The weights do not depend on the previous kernel: the first tile's
      // weight tiles are requested before waiting for it.
      int pre = 0;
      if ((int)blockIdx.x < num_tiles) {
        int mb, nb;
        tile_coords(blockIdx.x, num_m, num_n, mb, nb);
        pre = num_kb < C::STAGES ? num_kb : C::STAGES;
        for (int kb = 0; kb < pre; ++kb) {
          const uint32_t fb = full0 + 8 * kb;
          mbar_arrive_expect_tx(fb, tx);
          tma_load_2d(sB + kb * C::B_BYTES, &tmB, kb * BK, nb * BN, fb);
          if (DUAL) tma_load_2d(sB2 + kb * C::B_BYTES, &tmB2, kb * BK, nb * BN, fb);
        }
      }
      pdl_wait();
      bool first = true;
      for (int t = blockIdx.x; t < num_tiles; t += gridDim.x) {
        int mb, nb;
        tile_coords(t, num_m, num_n, mb, nb);
        bool ok = true;
        for (int kb = 0; kb < num_kb; ++kb) {
          const uint32_t fb = full0 + 8 * stage;
          if (first && kb < pre) {
            tma_load_2d(sA + stage * C::A_BYTES, &tmA, kb * BK, mb * BM, fb);
          } else {
            if (!mbar_wait_bounded(empty0 + 8 * stage, phase ^ 1, abort_flag, p.err, p.timeout_ns)) {
              ok = false;
              break;
            }
            mbar_arrive_expect_tx(fb, tx);
            tma_load_2d(sA + stage * C::A_BYTES, &tmA, kb * BK, mb * BM, fb);
            tma_load_2d(sB + stage * C::B_BYTES, &tmB, kb * BK, nb * BN, fb);
            if (DUAL) tma_load_2d(sB2 + stage * C::B_BYTES, &tmB2, kb * BK, nb * BN, fb);
          }
          ++issued;
          if (++stage == C::STAGES) { stage = 0; phase ^= 1; }
        }
        first = false;
        if (!ok) break;
      }
      // Drain: wait until the last copy issued into each stage has landed.
      for (int s = 0; s < C::STAGES; ++s) {
        if (issued <= s) break;
        const int64_t last = s + ((issued - 1 - s) / C::STAGES) * C::STAGES;
        mbar_wait_drain(full0 + 8 * s, (uint32_t)((last / C::STAGES) & 1), p.timeout_ns);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(BM, BN);
      int stage = 0;
      uint32_t phase = 0;
      int it = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < num_tiles && ok; t += gridDim.x, ++it) {
        const int acc = it & 1;
        if (!mbar_wait_bounded(tempty0 + 8 * acc, ((it >> 1) & 1) ^ 1, abort_flag, p.err,
                               p.timeout_ns)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * C::ACC_COLS;
        for (int kb = 0; kb < num_kb; ++kb) {
          if (!mbar_wait_bounded(full0 + 8 * stage, phase, abort_flag, p.err, p.timeout_ns)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_s = sA + stage * C::A_BYTES;
          const uint32_t b_s = sB + stage * C::B_BYTES;
#pragma unroll
          for (int k = 0; k < BK / UK; ++k) {
            const uint64_t ad = smem_desc_sw128(a_s + k * UK * 2);
            const uint64_t bd = smem_desc_sw128(b_s + k * UK * 2);
            const uint32_t accum = (kb > 0 || k > 0) ? 1u : 0u;
            tc_mma_f16(d_tmem, ad, bd, idesc, accum);
            if (DUAL) {
              const uint64_t b2d = smem_desc_sw128(sB2 + stage * C::B_BYTES + k * UK * 2);
              tc_mma_f16(d_tmem + BN, ad, b2d, idesc, accum);
            }
          }
          tc_commit(empty0 + 8 * stage);   // stage free once these MMAs have read it
          if (++stage == C::STAGES) { stage = 0; phase ^= 1; }
        }
        if (!ok) break;
        tc_commit(tfull0 + 8 * acc);       // accumulator ready for the epilogue
      }
      // Drain: every MMA issued by this thread has completed.
      tc_commit(drain);
      mbar_wait_drain(drain, 0, p.timeout_ns);
    }
  } else {
    // ------------------------------------------------------------ epilogue (warps 2..9)
    pdl_wait();
    const int quarter = warp & 3;   // TMEM lanes 32*quarter .. +31
    const int half = (warp - 2) >> 2;   // columns: chunks [half*NC/2, (half+1)*NC/2)
    const int row_in_tile = quarter * 32 + lane;
    int it = 0;
    for (int t = blockIdx.x; t < num_tiles; t += gridDim.x, ++it) {
      int mb, nb;
      tile_coords(t, num_m, num_n, mb, nb);
      const int acc = it & 1;
      int ok = 0;
      if (lane == 0)
        ok = mbar_wait_bounded(tfull0 + 8 * acc, (it >> 1) & 1, abort_flag, p.err, p.timeout_ns);
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) break;
      tc_fence_after();
      const uint32_t tacc = tmem_base + ((uint32_t)(quarter * 32) << 16) + acc * C::ACC_COLS;

      epilogue_tile<BN, DUAL, ROUTER>(p, tacc, mb * BM + row_in_tile, nb, half);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(tempty0 + 8 * acc);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, C::TMEM_COLS);
  }
}

// Two-CTA variant for large M (plain projections): a cluster of 2 CTAs owns
// a 256 x BN output tile. Each CTA stages its own 128 A rows and BN/2 of the
// weight rows (32 KB per stage for BN = 256, so 6 stages fit); one thread of
// the even CTA issues tcgen05.mma.cta_group::2 (M = 256), which reads both
// CTAs' shared memory and writes 128 accumulator rows into each CTA's TMEM.
// Stage completion is counted on the even CTA's full barriers (armed by the
// even CTA with both CTAs' bytes); MMA commits are multicast to the empty / accumulator-full barriers
// of both CTAs; both CTAs' epilogue warps release the accumulator on the even
// CTA's empty-accumulator barrier.
template <int BN, bool DUAL>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    gemm_tc2_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                    const __grid_constant__ CUtensorMap tmB2, const GemmDev p) {
  using C = TileCfg<BN, DUAL, true>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const uint32_t sA = smem_u32(smem);
  const uint32_t sB = sA + C::STAGES * C::A_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::STAGES * C::STAGE_BYTES);
  const uint32_t full0 = smem_u32(bars);
  const uint32_t empty0 = full0 + 8 * C::STAGES;
  const uint32_t tfull0 = empty0 + 8 * C::STAGES;
  const uint32_t tempty0 = tfull0 + 16;
  const uint32_t drain = tempty0 + 16;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * C::STAGES + 5);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  // weight tile of this CTA: plain -> rows [nb*BN + rank*BN/2, +BN/2) of W;
  // DUAL -> rows [nb*BN, +BN) of W (even CTA) or W2 (odd CTA)
  const CUtensorMap* tmW = (DUAL && rank == 1) ? &tmB2 : &tmB;
  const int brow_off = DUAL ? 0 : (int)rank * C::B_ROWS;
  const int pair = blockIdx.x >> 1;
  const int num_pairs = gridDim.x >> 1;
  const int num_m = (p.M + 2 * BM - 1) / (2 * BM);
  const int num_n = (p.N + BN - 1) / BN;
  const int num_tiles = num_m * num_n;
  const int num_kb = (p.K + BK - 1) / BK;

  pdl_trigger();
  if (threadIdx.x == 0) {
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(full0 + 8 * s, 1);              // the even CTA's producer arms both CTAs' bytes
      mbar_init(empty0 + 8 * s, 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(tfull0 + 8 * a, 1);
      mbar_init(tempty0 + 8 * a, 2 * kEpiWarps);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(tmW);
  }
  if (warp == 1) tmem_alloc_pair(smem_u32(tmem_slot), C::TMEM_COLS);
  tc_fence_before();
  cluster_sync();                 // both CTAs' barriers initialised, TMEM allocated
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const uint32_t full_lead = map_to_cta(full0, 0);
  const uint32_t tempty_lead = map_to_cta(tempty0, 0);

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer (both CTAs)
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int64_t issued = 0;
      // Only the even CTA arrives on (and arms) a stage's full barrier, with
      // both CTAs' bytes; the odd CTA's copies complete transactions on it,
      // possibly before it is armed (the transaction count may go negative).
      constexpr uint32_t tx = 2 * C::STAGE_BYTES;
      int pre = 0;
      if (pair < num_tiles) {
        int mb, nb;
        tile_coords(pair, num_m, num_n, mb, nb);
        pre = num_kb < C::STAGES ? num_kb : C::STAGES;
        for (int kb = 0; kb < pre; ++kb) {
          if (rank == 0) mbar_arrive_expect_tx(full0 + 8 * kb, tx);
          tma_load_2d_pair(sB + kb * C::B_BYTES, tmW, kb * BK, nb * BN + brow_off,
                           full_lead + 8 * kb);
        }
      }
      pdl_wait();
      bool first = true;
      for (int t = pair; t < num_tiles; t += num_pairs) {
        int mb, nb;
        tile_coords(t, num_m, num_n, mb, nb);
        const int arow0 = mb * 2 * BM + (int)rank * BM;
        const int brow0 = nb * BN + brow_off;
        bool ok = true;
        for (int kb = 0; kb < num_kb; ++kb) {
          const uint32_t fb = full_lead + 8 * stage;
          if (first && kb < pre) {
            tma_load_2d_pair(sA + stage * C::A_BYTES, &tmA, kb * BK, arow0, fb);
          } else {
            if (!mbar_wait_bounded(empty0 + 8 * stage, phase ^ 1, abort_flag, p.err, p.timeout_ns)) {
              ok = false;
              break;
            }
            if (rank == 0) mbar_arrive_expect_tx(full0 + 8 * stage, tx);
            tma_load_2d_pair(sA + stage * C::A_BYTES, &tmA, kb * BK, arow0, fb);
            tma_load_2d_pair(sB + stage * C::B_BYTES, tmW, kb * BK, brow0, fb);
          }
          ++issued;
          if (++stage == C::STAGES) { stage = 0; phase ^= 1; }
        }
        first = false;
        if (!ok) break;
      }
      // Drain (even CTA, whose full barriers count both CTAs' copies).
      if (rank == 0) {
        for (int s = 0; s < C::STAGES; ++s) {
          if (issued <= s) break;
          const int64_t last = s + ((issued - 1 - s) / C::STAGES) * C::STAGES;
          mbar_wait_drain(full0 + 8 * s, (uint32_t)((last / C::STAGES) & 1), p.timeout_ns);
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer (even CTA)
    if (lane == 0 && rank == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(2 * BM, DUAL ? 2 * BN : BN);
      int stage = 0;
      uint32_t phase = 0;
      int it = 0;
      bool ok = true;
      for (int t = pair; t < num_tiles && ok; t += num_pairs, ++it) {
        const int acc = it & 1;
        if (!mbar_wait_bounded(tempty0 + 8 * acc, ((it >> 1) & 1) ^ 1, abort_flag, p.err,
                               p.timeout_ns)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * C::ACC_COLS;
        for (int kb = 0; kb < num_kb; ++kb) {
          if (!mbar_wait_bounded(full0 + 8 * stage, phase, abort_flag, p.err, p.timeout_ns)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_s = sA + stage * C::A_BYTES;
          const uint32_t b_s = sB + stage * C::B_BYTES;
#pragma unroll
          for (int k = 0; k < BK / UK; ++k) {
            const uint64_t ad = smem_desc_sw128(a_s + k * UK * 2);
            const uint64_t bd = smem_desc_sw128(b_s + k * UK * 2);
            tc_mma_f16_pair(d_tmem, ad, bd, idesc, (kb > 0 || k > 0) ? 1u : 0u);
          }
          tc_commit_pair_multicast(empty0 + 8 * stage, 0x3);   // both CTAs' stage free
          if (++stage == C::STAGES) { stage = 0; phase ^= 1; }
        }
        if (!ok) break;
        tc_commit_pair_multicast(tfull0 + 8 * acc, 0x3);       // both CTAs' accumulators ready
      }
      tc_commit_pair_multicast(drain, 0x1);
      mbar_wait_drain(drain, 0, p.timeout_ns);
    }
  } else {
    // ------------------------------------------------------------ epilogue (warps 2..9, both CTAs)
    pdl_wait();
    const int quarter = warp & 3;
    const int half = (warp - 2) >> 2;
    const int row_in_tile = quarter * 32 + lane;
    int it = 0;
    for (int t = pair; t < num_tiles; t += num_pairs, ++it) {
      int mb, nb;
      tile_coords(t, num_m, num_n, mb, nb);
      const int acc = it & 1;
      int ok = 0;
      if (lane == 0)
        ok = mbar_wait_bounded(tfull0 + 8 * acc, (it >> 1) & 1, abort_flag, p.err, p.timeout_ns);
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) break;
      tc_fence_after();
      const uint32_t tacc = tmem_base + ((uint32_t)(quarter * 32) << 16) + acc * C::ACC_COLS;
      epilogue_tile<BN, DUAL, false>(p, tacc, mb * 2 * BM + (int)rank * BM + row_in_tile, nb, half);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(tempty_lead + 8 * acc);
    }
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync();                 // the pair's MMAs and copies are done before TMEM and smem go
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, C::TMEM_COLS);
  }
}

// ---------------------------------------------------------------- host side
}  // namespace

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  });
  return fn;
}

// Row-major bf16 [rows, cols] with leading dimension ld (elements): boxes of
// box_cols x box_rows with the 128-byte swizzle; out-of-range reads as zero.
bool make_tmap_bf16(CUtensorMap* m, const void* ptr, uint64_t rows, uint64_t cols, uint64_t ld,
                    uint32_t box_cols, uint32_t box_rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {ld * 2};
  cuuint32_t box[2] = {box_cols, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

namespace {

bool make_tmap(CUtensorMap* m, const void* ptr, uint64_t rows, uint64_t cols, uint64_t ld,
               uint32_t box_rows) {
  return make_tmap_bf16(m, ptr, rows, cols, ld, (uint32_t)BK, box_rows);
}

GemmDev make_dev(const GemmArgs& a, const Dev& dev) {
  GemmDev p;
  p.M = (int)a.M; p.N = a.N; p.K = a.K;
  p.act = a.epi.act;
  p.bias = static_cast<const bf16*>(a.epi.bias);
  p.add_packed = static_cast<const bf16*>(a.epi.add_packed); p.ld_add_packed = a.epi.ld_add_packed;
  p.add_rows = static_cast<const bf16*>(a.epi.add_rows); p.ld_add_rows = a.epi.ld_add_rows;
  p.rows = a.epi.rows;
  p.out_mapped = a.epi.out_mapped ? 1 : 0;
  p.out = static_cast<bf16*>(a.epi.out); p.ld_out = a.epi.ld_out;
  p.w2 = static_cast<const bf16*>(a.epi.w2); p.b2 = static_cast<const bf16*>(a.epi.b2);
  p.scores = a.epi.scores;
  p.rope_tab = a.epi.rope_tab;
  p.rope_pos = a.epi.rope_pos;
  p.rope_T = a.epi.rope_T;
  p.rope_half = a.epi.rope_half;
  p.rope_hd = a.epi.rope_hd;
  p.rope_cols = a.epi.rope_cols;
  p.vt = static_cast<bf16*>(a.epi.vt);
  p.vt_seq = a.epi.vt_seq;
  p.vt_pad = a.epi.vt_pad;
  p.vt_col0 = a.epi.vt_col0;
  p.vt_hd = a.epi.vt_hd;
  p.vt_hkv = a.epi.vt_hkv;
  p.err = dev.err;
  p.timeout_ns = kWaitTimeoutNs;
  return p;
}

template <int BN, bool DUAL, bool ROUTER>
cudaError_t launch(const GemmArgs& a, const Dev& dev) {
  using C = TileCfg<BN, DUAL>;
  static int attr_done[64] = {0};
  int device = 0;
  cudaGetDevice(&device);
  if (device < 64 && !attr_done[device]) {
    cudaError_t e = cudaFuncSetAttribute(gemm_tc_kernel<BN, DUAL, ROUTER>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM_BYTES);
    if (e != cudaSuccess) return e;
    attr_done[device] = 1;
  }
  CUtensorMap ta, tb, tb2;
  if (!make_tmap(&ta, a.A, (uint64_t)a.M, (uint64_t)a.K, (uint64_t)a.lda, BM) ||
      !make_tmap(&tb, a.W, (uint64_t)a.N, (uint64_t)a.K, (uint64_t)a.ldw, BN) ||
      (DUAL && !make_tmap(&tb2, a.W2, (uint64_t)a.N, (uint64_t)a.K, (uint64_t)a.ldw, BN)))
    return cudaErrorInvalidValue;
  if (!DUAL) tb2 = tb;
  GemmDev p = make_dev(a, dev);
  const int64_t num_tiles = ((a.M + BM - 1) / BM) * ((a.N + BN - 1) / BN);
  const int grid = (int)(num_tiles < dev.num_sms ? num_tiles : dev.num_sms);
  return launch_pdl(gemm_tc_kernel<BN, DUAL, ROUTER>, dim3(grid), dim3(kThreads), C::SMEM_BYTES,
                    dev.stream, ta, tb, tb2, p);
}

template <int BN, bool DUAL>
cudaError_t launch_pair(const GemmArgs& a, const Dev& dev) {
  using C = TileCfg<BN, DUAL, true>;
  static int attr_done[64] = {0};
  int device = 0;
  cudaGetDevice(&device);
  if (device < 64 && !attr_done[device]) {
    cudaError_t e = cudaFuncSetAttribute(gemm_tc2_kernel<BN, DUAL>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM_BYTES);
    if (e != cudaSuccess) return e;
    attr_done[device] = 1;
  }
  // A persistent grid must not exceed the CTA pairs that can be resident at
  // once (a TPC with one SM unavailable cannot host a pair).
  static int max_pairs[64] = {0};
  if (device < 64 && !max_pairs[device]) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(2 * (dev.num_sms / 2));
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = C::SMEM_BYTES;
    int n = 0;
    cudaError_t e = cudaOccupancyMaxActiveClusters(&n, gemm_tc2_kernel<BN, DUAL>, &cfg);
    if (e != cudaSuccess || n <= 0) return e != cudaSuccess ? e : cudaErrorInvalidConfiguration;
    max_pairs[device] = n;
  }
  const int64_t cap = device < 64 ? max_pairs[device] : dev.num_sms / 2;
  CUtensorMap ta, tb, tb2;
  if (!make_tmap(&ta, a.A, (uint64_t)a.M, (uint64_t)a.K, (uint64_t)a.lda, BM) ||
      !make_tmap(&tb, a.W, (uint64_t)a.N, (uint64_t)a.K, (uint64_t)a.ldw, C::B_ROWS) ||
      (DUAL && !make_tmap(&tb2, a.W2, (uint64_t)a.N, (uint64_t)a.K, (uint64_t)a.ldw, C::B_ROWS)))
    return cudaErrorInvalidValue;
  if (!DUAL) tb2 = tb;
  GemmDev p = make_dev(a, dev);
  const int64_t num_tiles = ((a.M + 2 * BM - 1) / (2 * BM)) * ((a.N + BN - 1) / BN);
  const int64_t pairs = num_tiles < cap ? num_tiles : cap;
  return launch_pdl(gemm_tc2_kernel<BN, DUAL>, dim3((unsigned)(2 * pairs)), dim3(kThreads),
                    C::SMEM_BYTES, dev.stream, ta, tb, tb2, p);
}

}  // namespace

cudaError_t gemm_bf16(const GemmArgs& a, const Dev& dev) {
  if (a.M <= 0) return cudaSuccess;
  if (a.epi.act == ACT_ROUTER) {
    if (a.N != 64) return cudaErrorInvalidValue;
    return launch<64, false, true>(a, dev);
  }
  // Large M: 256-row tiles on CTA pairs when that still gives every pair of
  // SMs at least two tiles (256 x 128 gate/up tiles for SwiGLU, 256 x 256
  // otherwise).
  if (a.epi.act == ACT_SWIGLU) {
    const int64_t pair_tiles = ((a.M + 255) / 256) * ((a.N + 127) / 128);
    if (a.N % 128 == 0 && pair_tiles >= dev.num_sms) return launch_pair<128, true>(a, dev);
    return launch<128, true, false>(a, dev);
  }
  const int64_t pair_tiles = ((a.M + 255) / 256) * ((a.N + 255) / 256);
  if (a.N % 256 == 0 && pair_tiles >= dev.num_sms) return launch_pair<256, false>(a, dev);
  // Pick the N tile that finishes in the fewest tile-time units: ceil(tiles /
  // SMs) waves, a 128-wide tile costing 0.58 of a 256-wide one (it moves 2/3
  // of the operand bytes for 1/2 of the flops).
  const int64_t mblocks = (a.M + BM - 1) / BM;
  const int64_t t256 = mblocks * ((a.N + 255) / 256);
  const int64_t t128 = mblocks * ((a.N + 127) / 128);
  const int64_t w256 = (t256 + dev.num_sms - 1) / dev.num_sms;
  const int64_t w128 = (t128 + dev.num_sms - 1) / dev.num_sms;
  if (a.N % 256 == 0 && 100 * w256 <= 58 * w128) return launch<256, false, false>(a, dev);
  return launch<128, false, false>(a, dev);
}

}  // namespace adadsf
