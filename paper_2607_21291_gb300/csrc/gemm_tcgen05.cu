// bf16 projections of the depth-sparse layer on the 5th-generation tensor cores.
//
// out = epilogue(A . W^T) with A [M, K] (packed kept tokens, row-major) and
// W [N, K] (nn.Linear layout); both operands are K-major, which is the layout
// tcgen05 reads natively. These are the dense contractions of Eqs. 1-2 (QKV,
// output and MLP projections).
//
// Kernel structure (one CTA per SM, 10 warps):
//   warp 0     TMA producer: 128x64 A tile and BNx64 W tile(s) per stage into a
//              STAGES-deep shared-memory ring, 128-byte swizzled, signalled
//              through mbarrier transaction counts.
//   warp 1     allocates TMEM; one thread issues tcgen05.mma (M=128, N=BN,
//              K=16, fp32 accumulator in TMEM) and commits stage releases and
//              accumulator hand-offs to mbarriers.
//   warps 2-9  epilogue: tcgen05.ld the accumulator (one row per thread, two
//              warps per 32-lane TMEM quarter splitting the columns), apply
//              bias / GELU / SwiGLU / rotary / residual / row scatter in
//              fp32, round once and store. Per-column constants (biases) are
//              staged in shared memory
//              and the first residual chunks loaded into registers before the
//              accumulator is ready, so their latency hides under the K loop.
//              GELU uses an erf with one exponential and no division (the
//              special-function unit bounds this epilogue).
// Three kernels share this structure:
//   gemm_tc_kernel     persistent, 128-row tiles; double-buffered TMEM so the
//                      epilogue of tile i runs under the main loop of tile i+1.
//   gemm_tc2_kernel    CTA pairs (cta_group::2), 256-row tiles, for large M.
//   gemm_tc_sk_kernel  small M: K split over the 2 or 4 CTAs of a cluster,
//                      partial tiles exchanged through a global scratch buffer.
// Two problem shapes beyond a single A . W^T:
//   two K sources      out = epi(A . W^T + A2 . W2^T): the K loop reads its
//                      first kb_split blocks through (A, W), the rest through
//                      (A2, W2) (the GPT-NeoX output and MLP-down projections
//                      of the parallel residual, Eq. 2, in one accumulator).
//   grouped            two independent problems (own A, W, epilogue) share one
//                      persistent launch (the GPT-NeoX QKV and MLP-up
//                      projections, which read the two norms of the same rows).
// Every barrier wait is bounded in time; on give-up the CTA records
// DEVERR_TIMEOUT, drains its in-flight copies and MMAs, frees TMEM and exits.
#include <cuda.h>
#include <cmath>
#include <cudaTypedefs.h>

#include <algorithm>
#include <cstdlib>
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
constexpr int kConstFloats = 256;   // staged per-column constants per epilogue warp and slot
constexpr int kStgBytes = 32 * 64;  // one 32-row x 32-column bf16 chunk per epilogue warp

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
  static constexpr int RING_BYTES = STAGES * STAGE_BYTES;
  static constexpr int ACC_COLS = BN * (DUAL ? 2 : 1);
  static constexpr int TMEM_COLS = 2 * ACC_COLS;
  static constexpr int BAR_BYTES = (2 * STAGES + 6) * 8 + 16;
  static constexpr int CONST_BYTES = kEpiWarps * 2 * kConstFloats * 4;
  static constexpr int STG_BYTES = kEpiWarps * kStgBytes;   // store staging, per epilogue warp
  static constexpr int SMEM_BYTES = RING_BYTES + 1024 + BAR_BYTES + CONST_BYTES + STG_BYTES;
  static_assert(TMEM_COLS == 128 || TMEM_COLS == 256 || TMEM_COLS == 512, "TMEM columns");
  static_assert(BAR_BYTES % 16 == 0, "constants stay 16-byte aligned");
  static_assert(SMEM_BYTES <= 232448, "shared memory");
};

struct GemmDev {
  int M, N, K;               // K: both sources together
  int bn;                    // tile width (N) of this problem's tiles
  int kb_split;              // k-blocks read through (tmA, tmB); the rest through (tmA2, tmB2)
  int act;
  const bf16* bias;
  const bf16* bias2;         // second bias (two K sources), or null
  const bf16* add; int64_t ld_add;   // residual: row m, or rows[m] when add_gathered
  int add_gathered;
  const int32_t* rows;
  int out_mapped;
  int a_box_rows;            // A rows a stage loads: 128, or fewer for a single block of fewer rows
  bf16* out; int64_t ld_out;
  // rotary embedding fused into the QKV epilogue (rope_tab == nullptr: off)
  const float2* rope_tab;    // [T][rope_half] (cos, sin)
  const int32_t* rope_pos;   // [M] original positions, or null: m % rope_T
  int rope_T, rope_half, rope_hd, rope_cols;
  bf16* vt;                  // transposed value heads (see Epilogue::vt)
  int vt_seq, vt_pad, vt_col0, vt_hd, vt_hkv;
  float* scratch;            // split-K partial tiles (gemm_tc_sk_kernel)
  // score gate: g = sigmoid(gate[rows[m]]); out = add + g v (add gathered) or
  // gbase + g (v + add - gbase) (add packed, gbase gathered)
  const float* gate;
  const bf16* gbase; int64_t ld_gbase;
  // folded RMSNorm of the A rows (see Epilogue::nrm_psum)
  const float* nrm_psum; const int32_t* nrm_rows; int nrm_nps; float nrm_inv_d, nrm_eps;
  const int32_t* a_gather;   // A rows by index (gemm_tc2_kernel; see GemmArgs::a_gather)
  // per-chunk sums of squares / Eq. 4 partials of the stored rows
  float* sq_out; int sq_ld;
  float4* cos_out; int cos_ld;
  const bf16* cin; int64_t ld_cin;
  float* out_f32;            // fp32 output instead of out (see Epilogue::out_f32)
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

__device__ __forceinline__ int tiles_of(const GemmDev& p, int bm) {
  return p.M > 0 ? ((p.M + bm - 1) / bm) * ((p.N + p.bn - 1) / p.bn) : 0;
}

// Tile t of a (possibly grouped) launch: problem, block coordinates, k-blocks.
struct TileInfo {
  int prob, mb, nb, nkb, kb_split, bn;
};
__device__ __forceinline__ TileInfo tile_info(int t, const GemmDev& p, const GemmDev& p2,
                                              int tiles0, int bm) {
  TileInfo ti;
  ti.prob = t < tiles0 ? 0 : 1;
  const GemmDev& P = ti.prob ? p2 : p;
  const int tt = ti.prob ? t - tiles0 : t;
  ti.bn = P.bn;
  tile_coords(tt, (P.M + bm - 1) / bm, (P.N + P.bn - 1) / P.bn, ti.mb, ti.nb);
  ti.nkb = (P.K + BK - 1) / BK;
  ti.kb_split = ti.prob ? 0 : P.kb_split;   // the second problem reads through (tmA2, tmB2)
  return ti;
}

// Tensor maps and K coordinate of k-block kb of a tile.
struct KbSrc {
  const CUtensorMap* a;
  const CUtensorMap* b;
  int kc;
};
__device__ __forceinline__ KbSrc kb_source(const TileInfo& ti, int kb, const CUtensorMap* tmA,
                                           const CUtensorMap* tmB, const CUtensorMap* tmA2,
                                           const CUtensorMap* tmB2) {
  const bool second = kb >= ti.kb_split;
  KbSrc s;
  s.a = second ? tmA2 : tmA;
  s.b = second ? tmB2 : tmB;
  s.kc = (second && ti.prob == 0 ? kb - ti.kb_split : kb) * BK;
  return s;
}

__device__ __forceinline__ float2 splat2(float a) { return make_float2(a, a); }

// erf(z) = 1 - exp(-z^2) R(z) for z >= 0 (erf is odd), R(z) = erfc(z) exp(z^2)
// approximated on [0, 4] by a degree-10 polynomial in z / 4 (coefficients
// and error bound from csrc/erf_poly.py: |error| <= 3.3e-7 in fp32); erf = 1
// beyond z = 4 (to 1.6e-8). One exponential, no division; two values at a
// time on the paired fp32 pipe (the epilogue is issue bound).
__device__ __forceinline__ float2 erf_fit2(float2 x) {
  const float zx = fminf(fabsf(x.x), 4.f), zy = fminf(fabsf(x.y), 4.f);
  const float2 u = make_float2(zx * 0.25f, zy * 0.25f);
  float2 r = splat2(1.019359436e+02f);
  r = __ffma2_rn(r, u, splat2(-3.950886841e+02f));
  r = __ffma2_rn(r, u, splat2(6.843880615e+02f));
  r = __ffma2_rn(r, u, splat2(-7.131018066e+02f));
  r = __ffma2_rn(r, u, splat2(5.127547607e+02f));
  r = __ffma2_rn(r, u, splat2(-2.798540955e+02f));
  r = __ffma2_rn(r, u, splat2(1.249815445e+02f));
  r = __ffma2_rn(r, u, splat2(-4.795371628e+01f));
  r = __ffma2_rn(r, u, splat2(1.599380779e+01f));
  r = __ffma2_rn(r, u, splat2(-4.513438225e+00f));
  r = __ffma2_rn(r, u, splat2(9.999998212e-01f));
  const float2 e = __ffma2_rn(make_float2(-__expf(-zx * zx), -__expf(-zy * zy)), r, splat2(1.f));
  return make_float2(copysignf(e.x, x.x), copysignf(e.y, x.y));
}
// exact GELU, 0.5 v (1 + erf(v / sqrt 2)), of two values
__device__ __forceinline__ float2 gelu2(float2 v) {
  const float2 e = erf_fit2(__fmul2_rn(v, splat2(0.70710678118654752f)));
  const float2 h = __fmul2_rn(v, splat2(0.5f));
  return __ffma2_rn(h, e, h);
}
// v sigmoid(v); the exponent is capped so the fast division stays in range.
__device__ __forceinline__ float silu_f(float v) {
  return v * __fdividef(1.f, 1.f + __expf(fminf(-v, 80.f)));
}

__device__ __forceinline__ void st_shared_f4(uint32_t addr, const float* f) {
  asm volatile("st.shared.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "f"(f[0]), "f"(f[1]),
               "f"(f[2]), "f"(f[3])
               : "memory");
}
__device__ __forceinline__ void ld_shared_f4(uint32_t addr, float* f) {
  asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(f[0]), "=f"(f[1]), "=f"(f[2]), "=f"(f[3])
               : "r"(addr)
               : "memory");
}

// Per-column constants of a tile, staged by each epilogue warp in its own
// shared-memory slot (no cross-warp barrier): sc[j] = bias[n] + bias2[n] for
// the tile's columns n = nb BN + j. Each lane moves 16 bytes at a time.
__device__ __forceinline__ void stage_consts(const GemmDev& p, int nb, int bn, uint32_t sc, int lane) {
  for (int j8 = lane; j8 < bn / 8; j8 += 32) {
    const int n = nb * bn + 8 * j8;
    float f[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    if (n < p.N) {
      if (p.bias) load_vec(p.bias + n, f);
      if (p.bias2) {
        float g[8];
        load_vec(p.bias2 + n, g);
#pragma unroll
        for (int i = 0; i < 8; ++i) f[i] += g[i];
      }
    }
    st_shared_f4(sc + 4u * (8 * j8), f);
    st_shared_f4(sc + 4u * (8 * j8 + 4), f + 4);
  }
  __syncwarp();
}

// v[0..31] += staged constants of columns [col, col + 32) of the tile.
__device__ __forceinline__ void add_consts32(uint32_t sc, int col, float* v) {
#pragma unroll
  for (int q = 0; q < 8; ++q) {
    float f[4];
    ld_shared_f4(sc + 4u * (col + 4 * q), f);
#pragma unroll
    for (int j = 0; j < 4; ++j) v[4 * q + j] += f[j];
  }
}

// Residual chunk: 32 bf16 of row rrow at column n0, as four 16-byte words.
__device__ __forceinline__ void load_res32(const GemmDev& p, int64_t rrow, int n0, uint4* u) {
  const uint4* src = reinterpret_cast<const uint4*>(p.add + rrow * p.ld_add + n0);
#pragma unroll
  for (int i = 0; i < 4; ++i) u[i] = src[i];
}

__device__ __forceinline__ void st_shared_u4(uint32_t addr, uint4 v) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
               : "memory");
}
__device__ __forceinline__ uint4 ld_shared_u4(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr)
               : "memory");
  return v;
}

// One 32-column bf16 chunk (4 x 16 bytes, pk) for each of the warp's 32
// rows (one per lane; dst = the lane's row at the chunk's first column, or
// null for no row), passed through the warp's staging area so that each
// global store instruction writes 8 rows x 64 contiguous bytes instead of
// 32 rows x 16 bytes (the rows are scattered or a full row apart). The 16-byte
// pieces are XOR-swizzled so neither phase has bank conflicts. Whole warp.
__device__ __forceinline__ void store_chunk_rows(uint32_t stg, int lane, const uint4* pk, bf16* dst) {
#pragma unroll
  for (int q = 0; q < 4; ++q) st_shared_u4(stg + lane * 64 + ((q ^ ((lane >> 1) & 3)) << 4), pk[q]);
  __syncwarp();
  const int q = lane & 3;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const int r = 8 * k + (lane >> 2);
    const uint4 v = ld_shared_u4(stg + r * 64 + ((q ^ ((r >> 1) & 3)) << 4));
    bf16* d = reinterpret_cast<bf16*>(
        __shfl_sync(0xffffffffu, (unsigned long long)reinterpret_cast<uintptr_t>(dst), r));
    if (d) *reinterpret_cast<uint4*>(d + 8 * q) = v;
  }
  __syncwarp();
}

// Store one 32-column chunk of output row orow (adding the residual `res`
// if RES and the problem has one); rows with !valid store nothing. Whole warp.
// EXTRA: the instance for the rarer epilogue features (score gate, chunk
// statistics for the next norm or Eq. 4); without it the plain residual path
// compiles as lean as possible.
template <bool RES, bool EXTRA>
__device__ __forceinline__ void epi_chunk_store(const GemmDev& p, float* v, const uint4* res,
                                                int64_t arow, int64_t orow, int n0, bool valid,
                                                uint32_t stg, int lane, int64_t m) {
  if (RES && p.add) {
    // the score gate of this row (gated variant)
    const float g = (EXTRA && p.gate && valid) ? 1.f / (1.f + expf(-p.gate[arow])) : 1.f;
    if (!EXTRA || !p.gate) {
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        float f[8];
        unpack16(res[i], f, bf16());
#pragma unroll
        for (int j = 0; j < 8; j += 2) {
          const float2 s2 = __fadd2_rn(make_float2(v[8 * i + j], v[8 * i + j + 1]), make_float2(f[j], f[j + 1]));
          v[8 * i + j] = s2.x;
          v[8 * i + j + 1] = s2.y;
        }
      }
    } else if (!p.gbase) {
      // gated, residual = the layer input x: out = x + g v
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        float f[8];
        unpack16(res[i], f, bf16());
#pragma unroll
        for (int j = 0; j < 8; ++j) v[8 * i + j] = fmaf(g, v[8 * i + j], f[j]);
      }
    } else {
      // gated, residual = h (packed), base = x: out = x + g (v + h - x)
      const uint4* gsrc = reinterpret_cast<const uint4*>(p.gbase + arow * p.ld_gbase + n0);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        float f[8], b[8];
        unpack16(res[i], f, bf16());
        unpack16(valid ? gsrc[i] : make_uint4(0, 0, 0, 0), b, bf16());
#pragma unroll
        for (int j = 0; j < 8; ++j) v[8 * i + j] = fmaf(g, (v[8 * i + j] + f[j]) - b[j], b[j]);
      }
    }
  }
  if (EXTRA && RES && valid && (p.sq_out || p.cos_out)) {
    // statistics of the chunk for the next norm / Eq. 4, from the fp32
    // values about to be stored (their bf16 rounding moves a sum of 32
    // squares by ~2^-9 relative at most)
    float sq = 0.f, dot = 0.f, nx = 0.f;
#pragma unroll
    for (int j = 0; j < 32; ++j) sq = fmaf(v[j], v[j], sq);
    if (p.cos_out) {
      // the layer input of this chunk: cos_in rows, else the residual
      const uint4* csrc = reinterpret_cast<const uint4*>(p.cin + arow * p.ld_cin + n0);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        float a[8];
        unpack16(p.cin ? csrc[i] : res[i], a, bf16());
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          dot = fmaf(a[j], v[8 * i + j], dot);
          nx = fmaf(a[j], a[j], nx);
        }
      }
    }
    if (p.sq_out) p.sq_out[m * p.sq_ld + (n0 >> 5)] = sq;
    if (p.cos_out) p.cos_out[m * p.cos_ld + (n0 >> 5)] = make_float4(dot, nx, sq, 0.f);
  }
  if (EXTRA && p.out_f32) {
    // fp32 output row chunk (uniform branch for the warp)
    if (valid) {
      float4* dst = reinterpret_cast<float4*>(p.out_f32 + orow * p.ld_out + n0);
#pragma unroll
      for (int i = 0; i < 8; ++i) dst[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
    }
    return;
  }
  uint4 pk[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) pk[i] = pack16(v + 8 * i, bf16());
  store_chunk_rows(stg, lane, pk, valid ? p.out + orow * p.ld_out + n0 : nullptr);
}

// Rotary halves of 32 or more features: chunk c (first half of a head's
// rotated features) and chunk c2 (second half) of row m: a' = a cos - b sin,
// b' = b cos + a sin. The row's (cos, sin) pairs are loaded 16 at a time (the
// first 16 of the tile may have been prefetched before the accumulator was
// ready: tpre), the accumulator 8 columns at a time. These are query / key
// columns: no activation, residual or transposed copy. SCALE: the
// accumulator is first multiplied by rs (the row's folded RMSNorm).
template <bool SCALE>
__device__ __forceinline__ void rope_pair(const GemmDev& p, uint32_t tacc, int c, int c2, int bn,
                                          int nb, uint32_t sc, bool has_consts,
                                          const float2* tab_row, bool mvalid, int64_t orow,
                                          const uint4 (&tpre)[2][4], bool use_pre, uint32_t stg,
                                          int lane, float rs) {
  const int n0 = nb * bn + c * 32, n2 = nb * bn + c2 * 32;
  const int i0 = n0 % p.rope_hd;
  uint4 pa[4], pb[4];   // the two chunks, bf16
#pragma unroll
  for (int gh = 0; gh < 2; ++gh) {
    float4 t[8];   // t[k] = (cos, sin) of features i0 + 16 gh + 2k and the next one
    if (mvalid) {
      const float4* t4 = reinterpret_cast<const float4*>(tab_row + i0 + 16 * gh);
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        if (gh == 0 && use_pre) {
          const uint4 q = tpre[k >> 2][k & 3];
          t[k] = make_float4(__uint_as_float(q.x), __uint_as_float(q.y), __uint_as_float(q.z),
                             __uint_as_float(q.w));
        } else {
          t[k] = t4[k];
        }
      }
    }
#pragma unroll
    for (int gg = 0; gg < 2; ++gg) {
      const int g = 2 * gh + gg;
      uint32_t ra[8], rb[8];
      tmem_ld8(tacc + c * 32 + 8 * g, ra);
      tmem_ld8(tacc + c2 * 32 + 8 * g, rb);
      tmem_ld_wait();
      float a[8], b[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        a[j] = __uint_as_float(ra[j]);
        b[j] = __uint_as_float(rb[j]);
        if (SCALE) {
          a[j] *= rs;
          b[j] *= rs;
        }
      }
      if (has_consts) {
        float f[4];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          ld_shared_f4(sc + 4u * (c * 32 + 8 * g + 4 * h), f);
#pragma unroll
          for (int j = 0; j < 4; ++j) a[4 * h + j] += f[j];
          ld_shared_f4(sc + 4u * (c2 * 32 + 8 * g + 4 * h), f);
#pragma unroll
          for (int j = 0; j < 4; ++j) b[4 * h + j] += f[j];
        }
      }
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const float4 q = t[4 * gg + j / 2];
        const float cs = (j & 1) ? q.z : q.x, sn = (j & 1) ? q.w : q.y;
        const float x = a[j], y = b[j];
        a[j] = x * cs - y * sn;
        b[j] = y * cs + x * sn;
      }
      pa[g] = pack16(a, bf16());
      pb[g] = pack16(b, bf16());
    }
  }
  store_chunk_rows(stg, lane, pa, mvalid ? p.out + orow * p.ld_out + n0 : nullptr);
  store_chunk_rows(stg, lane, pb, mvalid ? p.out + orow * p.ld_out + n2 : nullptr);
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

// Split-K partial tile of one CTA in global scratch: fp32, column groups of
// four outermost, [BN / 4][BM][4], so that a warp (32 consecutive rows) moves
// 512 contiguous bytes per 16-byte access.
__device__ __forceinline__ size_t partial_idx(int row, int col) {
  return (size_t)(col >> 2) * BM + row;   // in float4 units
}

// The partial tiles the epilogue adds (S == 0: none): those of the cluster's
// CTAs other than `rank`, in rank order, at base + q BM bn floats.
struct EpiRed {
  const float* base;
  int S, rank, bn;
};

// Values the epilogue fetched before the accumulator was ready.
// Rotary tiles (no residual) reuse the registers for the (cos, sin) pairs
// of their first chunk's first 16 features (res read as 8 float4).
struct EpiPre {
  uint4 res[2][4];   // residual of the first two chunks this warp finalises
  int n;             // how many of them are valid
  bool nt;           // res holds rotary pairs instead
  float rs;          // folded RMSNorm: the row's 1 / rms (1 without)
};

// The folded RMSNorm's scale of A row m from its chunk sums of squares
// (vector loads when the row of sums is 16-byte aligned); before the
// accumulator is ready.
__device__ __forceinline__ float norm_scale(const GemmDev& p, int m) {
  if (!p.nrm_psum || m >= p.M) return 1.f;
  const float* ps = p.nrm_psum + (int64_t)(p.nrm_rows ? p.nrm_rows[m] : m) * p.nrm_nps;
  float sum = 0.f;
  if ((p.nrm_nps & 3) == 0) {
    const float4* p4 = reinterpret_cast<const float4*>(ps);
    const int n4 = p.nrm_nps >> 2;
    float s0 = 0.f, s1 = 0.f;
    int i = 0;
    for (; i + 1 < n4; i += 2) {   // two vector loads in flight per step
      const float4 f = p4[i], h = p4[i + 1];
      s0 += (f.x + f.y) + (f.z + f.w);
      s1 += (h.x + h.y) + (h.z + h.w);
    }
    if (i < n4) {
      const float4 f = p4[i];
      s0 += (f.x + f.y) + (f.z + f.w);
    }
    sum = s0 + s1;
  } else {
    for (int i = 0; i < p.nrm_nps; ++i) sum += ps[i];
  }
  return 1.f / sqrtf(sum * p.nrm_inv_d + p.nrm_eps);
}

// Epilogue of one accumulator tile for the calling thread's row m over the
// chunks [c_lo, c_hi) of 32 TMEM columns -> constants / activation / rotary /
// residual / store. `sc` holds the staged
// per-column constants (has_consts), `pre` the prefetched residual chunks,
// `red` the split-K partial to add first. ROPE: the instance for rotary
// tiles (query / key / value projections, which have no residual).
template <int BN, bool DUAL, bool ROPE, bool EXTRA>
__device__ __forceinline__ void epilogue_tile(const GemmDev& p, uint32_t tacc, int m, int nb, int bn,
                                              int c_lo, int c_hi, uint32_t sc, bool has_consts,
                                              const EpiPre& pre, const EpiRed& red, uint32_t stg,
                                              int lane) {
  constexpr bool rope = ROPE && !DUAL;
  bool mvalid = m < p.M;
  int64_t arow = m;
  if (mvalid && p.rows) {
    arow = p.rows[m];
    if (arow < 0) mvalid = false;   // a row that bypasses the layer: nothing read or written
  }
  const int64_t orow = p.out_mapped ? arow : (int64_t)m;
  const float rs = pre.rs;   // folded RMSNorm of this A row (1 without)
  const float2* tab_row = nullptr;
  if (rope && mvalid)
    tab_row = p.rope_tab + (int64_t)(p.rope_pos ? p.rope_pos[m] : m % p.rope_T) * p.rope_half;
  const int row = m & (BM - 1);
#pragma unroll 1
  for (int c = c_lo; c < c_hi; ++c) {
    const int n0 = nb * bn + c * 32;
    // rotary halves of 32 or more features: chunk c pairs with chunk
    // c + half / 32, both handled by the owner of c
    const bool rot = rope && n0 < p.rope_cols;
    if (rot && p.rope_half >= 32) {
      if ((n0 % p.rope_hd) < p.rope_half && n0 < p.N)   // else done with its partner
        rope_pair<EXTRA>(p, tacc, c, c + p.rope_half / 32, bn, nb, sc, has_consts, tab_row, mvalid, orow,
                         pre.res, c == c_lo && pre.nt, stg, lane, rs);
      continue;
    }
    uint32_t r[32];
    uint32_t r2[DUAL ? 32 : 1];
    tmem_ld32(tacc + c * 32, r);
    if (DUAL) tmem_ld32(tacc + BN + c * 32, r2);
    tmem_ld_wait();
    if (n0 >= p.N) continue;   // (the same for the whole warp: the store below is warp-wide)
    float v[32];
#pragma unroll
    for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
    for (int q = 0; q < red.S; ++q) {
      if (q == red.rank) continue;
      const float4* src = reinterpret_cast<const float4*>(red.base + (size_t)q * BM * red.bn);
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const float4 f = __ldcg(src + partial_idx(row, c * 32 + 4 * j));
        v[4 * j] += f.x;
        v[4 * j + 1] += f.y;
        v[4 * j + 2] += f.z;
        v[4 * j + 3] += f.w;
      }
    }
    if (EXTRA && p.nrm_psum) {
#pragma unroll
      for (int j = 0; j < 32; ++j) v[j] *= rs;
    }
    if (has_consts) add_consts32(sc, c * 32, v);
    if (!DUAL && p.vt && n0 >= p.vt_col0 && mvalid) {
      // value columns: also store this row's 32 features transposed
      const int vc = n0 - p.vt_col0;
      const int bseq = m / p.vt_seq, j = m - bseq * p.vt_seq;
      bf16* dst = p.vt + ((int64_t)(bseq * p.vt_hkv + vc / p.vt_hd) * p.vt_hd + vc % p.vt_hd) *
                             p.vt_pad + j;
#pragma unroll
      for (int i = 0; i < 32; ++i) dst[(int64_t)i * p.vt_pad] = __float2bfloat16_rn(v[i]);
    }
    if (DUAL) {
#pragma unroll
      for (int j = 0; j < 32; ++j) v[j] = silu_f(v[j]) * ((EXTRA ? rs : 1.f) * __uint_as_float(r2[j]));
    } else if (p.act == ACT_GELU) {
#pragma unroll
      for (int j = 0; j < 32; j += 2) {
        const float2 g = gelu2(make_float2(v[j], v[j + 1]));
        v[j] = g.x;
        v[j + 1] = g.y;
      }
    }
    // residual of this chunk: prefetched for the first two, else loaded now
    uint4 res[4] = {make_uint4(0, 0, 0, 0), make_uint4(0, 0, 0, 0), make_uint4(0, 0, 0, 0),
                    make_uint4(0, 0, 0, 0)};
    if (!ROPE && p.add && mvalid) {
      const int k = c - c_lo;
      if (k < pre.n) {
#pragma unroll
        for (int i = 0; i < 4; ++i) res[i] = k == 0 ? pre.res[0][i] : pre.res[1][i];
      } else {
        load_res32(p, p.add_gathered ? arow : (int64_t)m, n0, res);
      }
    }
    if (rot && (n0 % p.rope_hd) == 0 && mvalid) {
      // rotary half of at most 16 features: both halves inside this chunk
      switch (p.rope_half) {
        case 4: rope_in_chunk<4>(v, tab_row); break;
        case 8: rope_in_chunk<8>(v, tab_row); break;
        case 16: rope_in_chunk<16>(v, tab_row); break;
        default: break;
      }
    }
    epi_chunk_store<!ROPE, EXTRA>(p, v, res, arow, orow, n0, mvalid, stg, lane, m);
  }
}

// Prefetch of the residual of chunks c_lo, c_lo + 1 for row m (before the
// accumulator is ready; the residual is an input of the kernel).
__device__ __forceinline__ void prefetch_res(const GemmDev& p, int m, int nb, int bn, int c_lo,
                                             int c_hi, EpiPre& pre) {
  pre.n = 0;
  if (!p.add || m >= p.M) return;
  const int64_t rrow = p.add_gathered ? (int64_t)p.rows[m] : (int64_t)m;
  if (rrow < 0) return;
  const int n = min(2, c_hi - c_lo);
  for (int k = 0; k < n; ++k) {
    const int n0 = nb * bn + (c_lo + k) * 32;
    if (n0 >= p.N) break;
    if (k == 0) load_res32(p, rrow, n0, pre.res[0]);
    else load_res32(p, rrow, n0, pre.res[1]);
    pre.n = k + 1;
  }
}

// The epilogue warps' part of a tile once its coordinates are known: stage
// constants, prefetch residuals, wait for the accumulator (bounded), run the
// epilogue. Returns false if the wait gave up.
template <int BN, bool DUAL, bool EXTRA>
__device__ __forceinline__ bool epilogue_role(const GemmDev& P, int m, int nb, int half,
                                              uint32_t tacc, uint32_t sc, uint32_t tfull,
                                              uint32_t parity, volatile int* abort_flag,
                                              int lane, uint32_t stg) {
  const int bn = P.bn;
  const int NC = bn / 32;
  const int c_lo = half * (NC / 2);
  const int c_hi = (half + 1) * (NC / 2);
  const bool has_consts = P.bias || P.bias2;
  if (has_consts) stage_consts(P, nb, bn, sc, lane);
  EpiPre pre;
  pre.n = 0;
  pre.nt = false;
  pre.rs = (EXTRA && P.nrm_psum) ? norm_scale(P, m) : 1.f;
  if (!P.rope_tab) {
    prefetch_res(P, m, nb, bn, c_lo, c_hi, pre);
  } else if (!DUAL && P.rope_half >= 32 && m < P.M) {
    // the first rotary chunk's (cos, sin) pairs (inputs of the kernel)
    const int n0 = nb * bn + c_lo * 32;
    if (n0 < P.rope_cols && n0 < P.N && (n0 % P.rope_hd) < P.rope_half) {
      const float4* t4 = reinterpret_cast<const float4*>(
          P.rope_tab + (int64_t)(P.rope_pos ? P.rope_pos[m] : m % P.rope_T) * P.rope_half + n0 % P.rope_hd);
      const uint4* q4 = reinterpret_cast<const uint4*>(t4);
#pragma unroll
      for (int k = 0; k < 8; ++k) pre.res[k >> 2][k & 3] = q4[k];
      pre.nt = true;
    }
  }
  int ok = 0;
  if (lane == 0) ok = mbar_wait_bounded(tfull, parity, abort_flag, P.err, P.timeout_ns);
  ok = __shfl_sync(0xffffffffu, ok, 0);
  if (!ok) return false;
  tc_fence_after();
  const EpiRed none = {nullptr, 0, 0, 0};
  if (!DUAL && P.rope_tab)
    epilogue_tile<BN, DUAL, true, EXTRA>(P, tacc, m, nb, bn, c_lo, c_hi, sc, has_consts, pre, none, stg, lane);
  else
    epilogue_tile<BN, DUAL, false, EXTRA>(P, tacc, m, nb, bn, c_lo, c_hi, sc, has_consts, pre, none, stg, lane);
  return true;
}

template <int BN, bool DUAL, bool EXTRA>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ CUtensorMap tmA2, const __grid_constant__ CUtensorMap tmB2,
                   const __grid_constant__ GemmDev p, const __grid_constant__ GemmDev p2) {
  using C = TileCfg<BN, DUAL>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const uint32_t sA = smem_u32(smem);
  const uint32_t sB = sA + C::STAGES * C::A_BYTES;
  const uint32_t sB2 = sB + C::STAGES * C::B_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::RING_BYTES);
  const uint32_t full0 = smem_u32(bars);
  const uint32_t empty0 = full0 + 8 * C::STAGES;
  const uint32_t tfull0 = empty0 + 8 * C::STAGES;
  const uint32_t tempty0 = tfull0 + 16;
  const uint32_t drain = tempty0 + 16;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * C::STAGES + 6);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const uint32_t sconst = sA + C::RING_BYTES + C::BAR_BYTES;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int tiles0 = tiles_of(p, BM);
  const int num_tiles = tiles0 + tiles_of(p2, BM);

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
    if (DUAL || p.kb_split * BK < p.K || p2.M > 0) {
      if (!DUAL) tma_prefetch_desc(&tmA2);
      tma_prefetch_desc(&tmB2);
    }
  }
  if (warp == 1) tmem_alloc(smem_u32(tmem_slot), C::TMEM_COLS);
  __syncwarp();
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
      // bytes per stage: the A tile and this problem's weight tile(s)
      auto stage_tx = [&](int bn) { return (uint32_t)(p.a_box_rows * BK * 2 + bn * BK * 2 * C::NUM_B); };
      // The weights do not depend on the previous kernel: the first tile's
      // weight tiles are requested before waiting for it.
      int pre = 0;
      if ((int)blockIdx.x < num_tiles) {
        const TileInfo ti = tile_info(blockIdx.x, p, p2, tiles0, BM);
        pre = ti.nkb < C::STAGES ? ti.nkb : C::STAGES;
        for (int kb = 0; kb < pre; ++kb) {
          const KbSrc src = kb_source(ti, kb, &tmA, &tmB, &tmA2, &tmB2);
          const uint32_t fb = full0 + 8 * kb;
          mbar_arrive_expect_tx(fb, stage_tx(ti.bn));
          tma_load_2d(sB + kb * C::B_BYTES, src.b, src.kc, ti.nb * ti.bn, fb);
          if (DUAL) tma_load_2d(sB2 + kb * C::B_BYTES, &tmB2, src.kc, ti.nb * ti.bn, fb);
        }
      }
      pdl_wait();
      bool first = true;
      for (int t = blockIdx.x; t < num_tiles; t += gridDim.x) {
        const TileInfo ti = tile_info(t, p, p2, tiles0, BM);
        const uint32_t tx = stage_tx(ti.bn);
        bool ok = true;
        for (int kb = 0; kb < ti.nkb; ++kb) {
          const KbSrc src = kb_source(ti, kb, &tmA, &tmB, &tmA2, &tmB2);
          const uint32_t fb = full0 + 8 * stage;
          if (first && kb < pre) {
            tma_load_2d(sA + stage * C::A_BYTES, src.a, src.kc, ti.mb * BM, fb);
          } else {
            if (!mbar_wait_bounded(empty0 + 8 * stage, phase ^ 1, abort_flag, p.err, p.timeout_ns)) {
              ok = false;
              break;
            }
            mbar_arrive_expect_tx(fb, tx);
            tma_load_2d(sA + stage * C::A_BYTES, src.a, src.kc, ti.mb * BM, fb);
            tma_load_2d(sB + stage * C::B_BYTES, src.b, src.kc, ti.nb * ti.bn, fb);
            if (DUAL) tma_load_2d(sB2 + stage * C::B_BYTES, &tmB2, src.kc, ti.nb * ti.bn, fb);
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
      constexpr uint32_t idesc_full = idesc_bf16_f32(BM, BN);
      constexpr uint32_t idesc_half = idesc_bf16_f32(BM, BN / 2 < 64 ? 64 : BN / 2);
      int stage = 0;
      uint32_t phase = 0;
      int it = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < num_tiles && ok; t += gridDim.x, ++it) {
        const TileInfo ti = tile_info(t, p, p2, tiles0, BM);
        const uint32_t idesc = ti.bn == BN ? idesc_full : idesc_half;
        const int acc = it & 1;
        if (!mbar_wait_bounded(tempty0 + 8 * acc, ((it >> 1) & 1) ^ 1, abort_flag, p.err,
                               p.timeout_ns)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * C::ACC_COLS;
        for (int kb = 0; kb < ti.nkb; ++kb) {
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
      const TileInfo ti = tile_info(t, p, p2, tiles0, BM);
      const GemmDev& P = ti.prob ? p2 : p;
      const int acc = it & 1;
      const uint32_t sc = sconst + 4u * kConstFloats * ((warp - 2) * 2 + acc);
      const uint32_t tacc = tmem_base + ((uint32_t)(quarter * 32) << 16) + acc * C::ACC_COLS;
      if (!epilogue_role<BN, DUAL, EXTRA>(P, ti.mb * BM + row_in_tile, ti.nb, half, tacc, sc,
                                           tfull0 + 8 * acc, (it >> 1) & 1, abort_flag, lane,
                                           sconst + C::CONST_BYTES + kStgBytes * (warp - 2)))
        break;
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(tempty0 + 8 * acc);
    }
  }

  // Reconverge each warp first: in the producer and MMA warps only lane 0
  // ran the role loop, and the block barrier counts whole warps.
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, C::TMEM_COLS);
  }
}

// Split-K variant for GEMMs with too few output tiles to fill the GPU (small
// M): a cluster of S CTAs (S = 2 or 4, consecutive along x) owns one 128 x BN
// output tile; CTA r accumulates k-blocks [r KB/S, (r+1) KB/S) in its own
// TMEM and finalises the columns [r W, (r+1) W), W = BN / S. Reduce-scatter
// through the L2: each CTA writes its partial of the other CTAs' columns to
// its slot of a global scratch buffer, a cluster barrier (release / acquire)
// orders the writes before the reads, and each CTA adds the other CTAs'
// slots in rank order (a fixed order: the sum does not depend on timing) to
// its own columns before the usual epilogue.
template <int BN, bool EXTRA>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_tc_sk_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                      const __grid_constant__ CUtensorMap tmA2, const __grid_constant__ CUtensorMap tmB2,
                      const __grid_constant__ GemmDev p) {
  using C = TileCfg<BN, false>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const uint32_t sA = smem_u32(smem);
  const uint32_t sB = sA + C::STAGES * C::A_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::RING_BYTES);
  const uint32_t full0 = smem_u32(bars);
  const uint32_t empty0 = full0 + 8 * C::STAGES;
  const uint32_t tfull = empty0 + 8 * C::STAGES;
  const uint32_t drain = tfull + 8;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * C::STAGES + 6);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const uint32_t sconst = sA + C::RING_BYTES + C::BAR_BYTES;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int S = (int)cluster_nctarank();
  const int rank = (int)cluster_ctarank();
  const int NCO = BN / S / 32;                // chunks finalised by each CTA
  const int tile = blockIdx.x / S;
  const TileInfo ti = tile_info(tile, p, p, 1 << 30, BM);
  const int kb0 = rank * ti.nkb / S;
  const int kb1 = (rank + 1) * ti.nkb / S;
  const int nkb = kb1 - kb0;

  pdl_trigger();
  if (threadIdx.x == 0) {
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    mbar_init(tfull, 1);
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_barrier_init();
    fence_proxy_async_smem();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
    if (p.kb_split < ti.nkb) {
      tma_prefetch_desc(&tmA2);
      tma_prefetch_desc(&tmB2);
    }
  }
  if (warp == 1) tmem_alloc(smem_u32(tmem_slot), BN);
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  // epilogue warps: this warp's TMEM lane quarter, its chunks of a CTA's
  // columns (both halves when there are two or more chunks, else half 0)
  const int quarter = warp & 3;
  const int half = (warp - 2) >> 2;
  const int row = quarter * 32 + lane;
  const int m = ti.mb * BM + row;
  const uint32_t tacc = tmem_base + ((uint32_t)(quarter * 32) << 16);
  const uint32_t sc = sconst + 4u * kConstFloats * ((warp - 2) * 2);
  const int h_lo = NCO >= 2 ? half * (NCO / 2) : half;
  const int h_hi = NCO >= 2 ? (half + 1) * (NCO / 2) : 1;
  const int c_lo = rank * NCO + h_lo, c_hi = rank * NCO + h_hi;
  const bool has_consts = p.bias || p.bias2;
  EpiPre pre;
  pre.n = 0;
  pre.nt = false;
  pre.rs = 1.f;
  int ok = 0;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      const uint32_t tx = (uint32_t)(p.a_box_rows * BK * 2 + C::B_BYTES);
      const int npre = nkb < C::STAGES ? nkb : C::STAGES;
      for (int i = 0; i < npre; ++i) {   // weights first: independent of the previous kernel
        const KbSrc src = kb_source(ti, kb0 + i, &tmA, &tmB, &tmA2, &tmB2);
        mbar_arrive_expect_tx(full0 + 8 * i, tx);
        tma_load_2d(sB + i * C::B_BYTES, src.b, src.kc, ti.nb * BN, full0 + 8 * i);
      }
      pdl_wait();
      int stage = 0;
      uint32_t phase = 0;
      int issued = 0;
      for (int i = 0; i < nkb; ++i) {
        const KbSrc src = kb_source(ti, kb0 + i, &tmA, &tmB, &tmA2, &tmB2);
        const uint32_t fb = full0 + 8 * stage;
        if (i < npre) {
          tma_load_2d(sA + stage * C::A_BYTES, src.a, src.kc, ti.mb * BM, fb);
        } else {
          if (!mbar_wait_bounded(empty0 + 8 * stage, phase ^ 1, abort_flag, p.err, p.timeout_ns))
            break;
          mbar_arrive_expect_tx(fb, tx);
          tma_load_2d(sA + stage * C::A_BYTES, src.a, src.kc, ti.mb * BM, fb);
          tma_load_2d(sB + stage * C::B_BYTES, src.b, src.kc, ti.nb * BN, fb);
        }
        ++issued;
        if (++stage == C::STAGES) { stage = 0; phase ^= 1; }
      }
      for (int s = 0; s < C::STAGES; ++s) {
        if (issued <= s) break;
        const int last = s + ((issued - 1 - s) / C::STAGES) * C::STAGES;
        mbar_wait_drain(full0 + 8 * s, (uint32_t)((last / C::STAGES) & 1), p.timeout_ns);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(BM, BN);
      int stage = 0;
      uint32_t phase = 0;
      bool mok = true;
      for (int i = 0; i < nkb; ++i) {
        if (!mbar_wait_bounded(full0 + 8 * stage, phase, abort_flag, p.err, p.timeout_ns)) {
          mok = false;
          break;
        }
        tc_fence_after();
        const uint32_t a_s = sA + stage * C::A_BYTES;
        const uint32_t b_s = sB + stage * C::B_BYTES;
#pragma unroll
        for (int k = 0; k < BK / UK; ++k) {
          const uint64_t ad = smem_desc_sw128(a_s + k * UK * 2);
          const uint64_t bd = smem_desc_sw128(b_s + k * UK * 2);
          tc_mma_f16(tmem_base, ad, bd, idesc, (i > 0 || k > 0) ? 1u : 0u);
        }
        tc_commit(empty0 + 8 * stage);
        if (++stage == C::STAGES) { stage = 0; phase ^= 1; }
      }
      if (mok) tc_commit(tfull);
      tc_commit(drain);
      mbar_wait_drain(drain, 0, p.timeout_ns);
    }
  } else {
    // ------------------------------------------------------------ epilogue, part 1
    pdl_wait();
    if (has_consts) stage_consts(p, ti.nb, BN, sc, lane);
    if (lane == 0) ok = mbar_wait_bounded(tfull, 0, abort_flag, p.err, p.timeout_ns);
    ok = __shfl_sync(0xffffffffu, ok, 0);
    tc_fence_after();
    if (ok) {
      // this CTA's partial of the other CTAs' columns -> its scratch slot
      float4* dst = reinterpret_cast<float4*>(p.scratch + (size_t)blockIdx.x * BM * BN);
      for (int q = 0; q < S; ++q) {
        if (q == rank) continue;
        for (int c = q * NCO + h_lo; c < q * NCO + h_hi; ++c) {
          uint32_t r[32];
          tmem_ld32(tacc + c * 32, r);
          tmem_ld_wait();
#pragma unroll
          for (int j = 0; j < 8; ++j)
            __stcg(dst + partial_idx(row, c * 32 + 4 * j),
                   make_float4(__uint_as_float(r[4 * j]), __uint_as_float(r[4 * j + 1]),
                               __uint_as_float(r[4 * j + 2]), __uint_as_float(r[4 * j + 3])));
        }
      }
      if (h_lo < h_hi) {
        prefetch_res(p, m, ti.nb, BN, c_lo, c_hi, pre);
        if (EXTRA && p.nrm_psum) pre.rs = norm_scale(p, m);
      }
    }
  }

  // Every CTA's partials are in the scratch buffer (release / acquire at
  // cluster scope); a CTA that gave up still arrives.
  __syncwarp();
  cluster_sync();

  if (warp >= 2 && ok && h_lo < h_hi) {
    // ------------------------------------------------------------ epilogue, part 2
    const EpiRed red = {p.scratch + (size_t)tile * S * BM * BN, S, rank, BN};
    const uint32_t stg = sconst + C::CONST_BYTES + kStgBytes * (warp - 2);
    if (p.rope_tab)   // rotary halves of at most 16 features (one chunk)
      epilogue_tile<BN, false, true, EXTRA>(p, tacc, m, ti.nb, BN, c_lo, c_hi, sc, has_consts, pre, red, stg,
                                            lane);
    else
      epilogue_tile<BN, false, false, EXTRA>(p, tacc, m, ti.nb, BN, c_lo, c_hi, sc, has_consts, pre, red, stg,
                                             lane);
  }

  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, BN);
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
// CTA's empty-accumulator barrier. Two K sources and grouped problems work
// as in the one-CTA kernel (not with DUAL).
template <int BN, bool DUAL, bool EXTRA>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    gemm_tc2_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                    const __grid_constant__ CUtensorMap tmA2, const __grid_constant__ CUtensorMap tmB2,
                    const __grid_constant__ GemmDev p, const __grid_constant__ GemmDev p2) {
  using C = TileCfg<BN, DUAL, true>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const uint32_t sA = smem_u32(smem);
  const uint32_t sB = sA + C::STAGES * C::A_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::RING_BYTES);
  const uint32_t full0 = smem_u32(bars);
  const uint32_t empty0 = full0 + 8 * C::STAGES;
  const uint32_t tfull0 = empty0 + 8 * C::STAGES;
  const uint32_t tempty0 = tfull0 + 16;
  const uint32_t drain = tempty0 + 16;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * C::STAGES + 6);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const uint32_t sconst = sA + C::RING_BYTES + C::BAR_BYTES;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  // weight tile of this CTA: plain -> rows [nb*BN + rank*BN/2, +BN/2) of W;
  // DUAL -> rows [nb*BN, +BN) of W (even CTA) or W2 (odd CTA)
  const int brow_off = DUAL ? 0 : (int)rank * C::B_ROWS;
  const int pair = blockIdx.x >> 1;
  const int num_pairs = gridDim.x >> 1;
  const int tiles0 = tiles_of(p, 2 * BM);
  const int num_tiles = tiles0 + tiles_of(p2, 2 * BM);
  // DUAL: the odd CTA reads the second weight for every k-block
  auto wmap = [&](const KbSrc& s) -> const CUtensorMap* {
    return DUAL ? (rank == 1 ? &tmB2 : &tmB) : s.b;
  };

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
    tma_prefetch_desc(&tmB);
    if (DUAL || p.kb_split * BK < p.K || p2.M > 0) {
      if (!DUAL) tma_prefetch_desc(&tmA2);
      tma_prefetch_desc(&tmB2);
    }
  }
  if (warp == 1) tmem_alloc_pair(smem_u32(tmem_slot), C::TMEM_COLS);
  __syncwarp();
  tc_fence_before();
  cluster_sync();                 // both CTAs' barriers initialised, TMEM allocated
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const uint32_t full_lead = map_to_cta(full0, 0);
  const uint32_t tempty_lead = map_to_cta(tempty0, 0);

  if (warp == 0 && p.a_gather) {
    // ------------------------------------------------------------ TMA producer, gathered A
    // (one problem, one K source). Lane l brings rows 4l .. 4l + 3 of the
    // CTA's 128-row block, row r of the block being row a_gather[r] of A, by
    // one row gather per k-block; lane 0 waits for the stage and loads the
    // weight tile. Rows past M repeat the last one (never stored).
    int stage = 0;
    uint32_t phase = 0;
    int64_t issued = 0;
    constexpr uint32_t tx = 2 * C::STAGE_BYTES;
    int pre = 0;
    if (pair < num_tiles) {
      const TileInfo ti = tile_info(pair, p, p2, tiles0, 2 * BM);
      pre = ti.nkb < C::STAGES ? ti.nkb : C::STAGES;
      if (lane == 0) {
        for (int kb = 0; kb < pre; ++kb) {
          if (rank == 0) mbar_arrive_expect_tx(full0 + 8 * kb, tx);
          tma_load_2d_pair(sB + kb * C::B_BYTES, &tmB, kb * BK, ti.nb * BN + brow_off, full_lead + 8 * kb);
        }
      }
    }
    pdl_wait();
    bool first = true;
    for (int t = pair; t < num_tiles; t += num_pairs) {
      const TileInfo ti = tile_info(t, p, p2, tiles0, 2 * BM);
      const int m0 = ti.mb * 2 * BM + (int)rank * BM + 4 * lane;
      int g[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) g[j] = __ldg(p.a_gather + min(m0 + j, p.M - 1));
      const int brow0 = ti.nb * BN + brow_off;
      bool ok = true;
      for (int kb = 0; kb < ti.nkb; ++kb) {
        const uint32_t fb = full_lead + 8 * stage;
        if (!(first && kb < pre)) {
          int w = 1;
          if (lane == 0) {
            w = mbar_wait_bounded(empty0 + 8 * stage, phase ^ 1, abort_flag, p.err, p.timeout_ns);
            if (w) {
              if (rank == 0) mbar_arrive_expect_tx(full0 + 8 * stage, tx);
              tma_load_2d_pair(sB + stage * C::B_BYTES, &tmB, kb * BK, brow0, fb);
            }
          }
          ok = __shfl_sync(0xffffffffu, w, 0) != 0;
          if (!ok) break;
        }
        tma_gather4_pair(sA + stage * C::A_BYTES + lane * 4 * BK * 2, &tmA, kb * BK, g[0], g[1], g[2], g[3], fb);
        ++issued;
        if (++stage == C::STAGES) { stage = 0; phase ^= 1; }
      }
      first = false;
      if (!ok) break;
    }
    // Drain (even CTA, whose full barriers count both CTAs' copies).
    if (lane == 0 && rank == 0) {
      for (int s = 0; s < C::STAGES; ++s) {
        if (issued <= s) break;
        const int64_t last = s + ((issued - 1 - s) / C::STAGES) * C::STAGES;
        mbar_wait_drain(full0 + 8 * s, (uint32_t)((last / C::STAGES) & 1), p.timeout_ns);
      }
    }
  } else if (warp == 0) {
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
        const TileInfo ti = tile_info(pair, p, p2, tiles0, 2 * BM);
        pre = ti.nkb < C::STAGES ? ti.nkb : C::STAGES;
        for (int kb = 0; kb < pre; ++kb) {
          const KbSrc src = kb_source(ti, kb, &tmA, &tmB, &tmA2, &tmB2);
          if (rank == 0) mbar_arrive_expect_tx(full0 + 8 * kb, tx);
          tma_load_2d_pair(sB + kb * C::B_BYTES, wmap(src), src.kc, ti.nb * BN + brow_off,
                           full_lead + 8 * kb);
        }
      }
      pdl_wait();
      bool first = true;
      for (int t = pair; t < num_tiles; t += num_pairs) {
        const TileInfo ti = tile_info(t, p, p2, tiles0, 2 * BM);
        const int arow0 = ti.mb * 2 * BM + (int)rank * BM;
        const int brow0 = ti.nb * BN + brow_off;
        bool ok = true;
        for (int kb = 0; kb < ti.nkb; ++kb) {
          const KbSrc src = kb_source(ti, kb, &tmA, &tmB, &tmA2, &tmB2);
          const uint32_t fb = full_lead + 8 * stage;
          if (first && kb < pre) {
            tma_load_2d_pair(sA + stage * C::A_BYTES, src.a, src.kc, arow0, fb);
          } else {
            if (!mbar_wait_bounded(empty0 + 8 * stage, phase ^ 1, abort_flag, p.err, p.timeout_ns)) {
              ok = false;
              break;
            }
            if (rank == 0) mbar_arrive_expect_tx(full0 + 8 * stage, tx);
            tma_load_2d_pair(sA + stage * C::A_BYTES, src.a, src.kc, arow0, fb);
            tma_load_2d_pair(sB + stage * C::B_BYTES, wmap(src), src.kc, brow0, fb);
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
        const TileInfo ti = tile_info(t, p, p2, tiles0, 2 * BM);
        const int acc = it & 1;
        if (!mbar_wait_bounded(tempty0 + 8 * acc, ((it >> 1) & 1) ^ 1, abort_flag, p.err,
                               p.timeout_ns)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * C::ACC_COLS;
        for (int kb = 0; kb < ti.nkb; ++kb) {
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
      const TileInfo ti = tile_info(t, p, p2, tiles0, 2 * BM);
      const GemmDev& P = ti.prob ? p2 : p;
      const int acc = it & 1;
      const uint32_t sc = sconst + 4u * kConstFloats * ((warp - 2) * 2 + acc);
      const uint32_t tacc = tmem_base + ((uint32_t)(quarter * 32) << 16) + acc * C::ACC_COLS;
      if (!epilogue_role<BN, DUAL, EXTRA>(P, ti.mb * 2 * BM + (int)rank * BM + row_in_tile, ti.nb,
                                          half, tacc, sc, tfull0 + 8 * acc, (it >> 1) & 1,
                                          abort_flag, lane, sconst + C::CONST_BYTES + kStgBytes * (warp - 2)))
        break;
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(tempty_lead + 8 * acc);
    }
  }

  // Reconverge each warp first: in the producer and MMA warps only lane 0
  // ran the role loop, and the block barrier counts whole warps.
  __syncwarp();
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

bool make_dev(const GemmArgs& a, const Dev& dev, GemmDev& p) {
  p = GemmDev{};
  if (a.epi.add_packed && a.epi.add_rows) return false;   // one residual source per launch
  if (a.epi.rope_tab && (a.epi.add_packed || a.epi.add_rows)) return false;   // rotary tiles: none
  if (a.K2 > 0 && a.K % BK != 0) return false;            // the K sources meet on a k-block
  p.M = (int)a.M; p.N = a.N; p.K = a.K + (a.K2 > 0 ? a.K2 : 0);
  p.kb_split = a.K2 > 0 ? a.K / BK : (p.K + BK - 1) / BK;
  p.act = a.epi.act;
  p.bias = static_cast<const bf16*>(a.epi.bias);
  p.bias2 = static_cast<const bf16*>(a.epi.bias2);
  if (a.epi.add_packed) {
    p.add = static_cast<const bf16*>(a.epi.add_packed);
    p.ld_add = a.epi.ld_add_packed;
    p.add_gathered = 0;
  } else if (a.epi.add_rows) {
    p.add = static_cast<const bf16*>(a.epi.add_rows);
    p.ld_add = a.epi.ld_add_rows;
    p.add_gathered = a.epi.rows ? 1 : 0;
  }
  p.rows = a.epi.rows;
  p.a_gather = a.a_gather;
  p.out_mapped = a.epi.out_mapped ? 1 : 0;
  p.out = static_cast<bf16*>(a.epi.out); p.ld_out = a.epi.ld_out;
  if (a.epi.nrm_psum) {
    if (a.epi.nrm_d <= 0 || a.epi.nrm_nps <= 0) return false;
    p.nrm_psum = a.epi.nrm_psum;
    p.nrm_rows = a.epi.nrm_rows;
    p.nrm_nps = a.epi.nrm_nps;
    p.nrm_inv_d = 1.f / (float)a.epi.nrm_d;
    p.nrm_eps = a.epi.nrm_eps;
  }
  if (a.epi.sq_out || a.epi.cos_out) {
    // statistics of stored rows: plain or residual outputs, no rotary tiles
    if (a.epi.rope_tab || a.N % 32 != 0) return false;
    if (a.epi.cos_out && !a.epi.cos_in && !a.epi.add_rows) return false;
    p.sq_out = a.epi.sq_out;
    p.sq_ld = a.epi.sq_ld;
    p.cos_out = a.epi.cos_out;
    p.cos_ld = a.epi.cos_ld;
    p.cin = static_cast<const bf16*>(a.epi.cos_in);
    p.ld_cin = a.epi.ld_cos_in;
  }
  if (a.epi.out_f32) {
    if (a.epi.rope_tab || a.epi.add_packed || a.epi.add_rows || a.epi.vt || a.N % 32 != 0) return false;
    p.out_f32 = a.epi.out_f32;
  }
  if (a.epi.gate_scores) {
    // gated residual: x gathered (out = x + g v), or h packed with x as the base
    if (a.epi.rope_tab) return false;
    if (a.epi.gate_base ? !a.epi.add_packed : !a.epi.add_rows) return false;
    p.gate = a.epi.gate_scores;
    p.gbase = static_cast<const bf16*>(a.epi.gate_base);
    p.ld_gbase = a.epi.ld_gate_base;
  }
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
  p.scratch = a.scratch;
  p.err = dev.err;
  p.timeout_ns = kWaitTimeoutNs;
  return true;
}

// Tensor maps of one problem: (A, W) and, for two K sources, (A2, W2).
bool problem_maps(const GemmArgs& a, uint32_t a_rows, uint32_t b_rows, CUtensorMap& ta,
                  CUtensorMap& tb, CUtensorMap* ta2, CUtensorMap* tb2) {
  // gathered A: all of A's rows, boxes one row high (four per gather)
  if (!(a.a_gather ? make_tmap(&ta, a.A, (uint64_t)a.a_gather_rows, (uint64_t)a.K, (uint64_t)a.lda, 1)
                   : make_tmap(&ta, a.A, (uint64_t)a.M, (uint64_t)a.K, (uint64_t)a.lda, a_rows)) ||
      !make_tmap(&tb, a.W, (uint64_t)a.N, (uint64_t)a.K, (uint64_t)a.ldw, b_rows))
    return false;
  if (a.K2 > 0) {
    if (!ta2 || !tb2 ||
        !make_tmap(ta2, a.A2, (uint64_t)a.M, (uint64_t)a.K2, (uint64_t)a.lda2, a_rows) ||
        !make_tmap(tb2, a.Wk2, (uint64_t)a.N, (uint64_t)a.K2, (uint64_t)a.ldwk2, b_rows))
      return false;
  }
  return true;
}

// Maps and device descriptors for a launch of problem `a` (plus the grouped
// problem `b`, or the DUAL second weight). bn: the kernel's tile width; a
// problem may ask for half of it (tile_n); b_rows: weight rows a CTA stages
// per full-width tile (half of bn on CTA pairs).
template <bool DUAL>
cudaError_t prepare(const GemmArgs& a, const GemmArgs* b, uint32_t a_rows, int bn, uint32_t b_rows,
                    const Dev& dev, CUtensorMap (&tm)[4], GemmDev& p, GemmDev& p2) {
  auto width = [&](const GemmArgs& g) { return g.tile_n > 0 && g.tile_n < bn ? g.tile_n : bn; };
  auto rows = [&](const GemmArgs& g) { return (uint32_t)((uint64_t)b_rows * width(g) / bn); };
  if ((a.tile_n && width(a) * 2 != bn && width(a) != bn) || (b && b->tile_n && width(*b) * 2 != bn && width(*b) != bn))
    return cudaErrorInvalidValue;
  if (!make_dev(a, dev, p)) return cudaErrorInvalidValue;
  p.bn = width(a);
  p.a_box_rows = (int)a_rows;
  p2 = GemmDev{};
  p2.bn = bn;
  p2.a_box_rows = (int)a_rows;
  if (!problem_maps(a, a_rows, rows(a), tm[0], tm[1], &tm[2], &tm[3])) return cudaErrorInvalidValue;
  if (DUAL) {
    if (p.bn != bn || !make_tmap(&tm[3], a.W2, (uint64_t)a.N, (uint64_t)a.K, (uint64_t)a.ldw, b_rows))
      return cudaErrorInvalidValue;
    tm[2] = tm[0];
  } else if (b) {
    if (a.K2 > 0 || b->K2 > 0 || !make_dev(*b, dev, p2)) return cudaErrorInvalidValue;
    p2.bn = width(*b);
    p2.a_box_rows = (int)a_rows;
    if (!problem_maps(*b, a_rows, rows(*b), tm[2], tm[3], nullptr, nullptr))
      return cudaErrorInvalidValue;
  } else if (a.K2 == 0) {
    tm[2] = tm[0];
    tm[3] = tm[1];
  }
  return cudaSuccess;
}

// A rows a stage of the one-CTA kernels loads. A single block of fewer than
// 128 rows (a decode step's few rows) loads only those, rounded up to 8:
// the rows past them stay as they are in shared memory, and the
// accumulator rows they give are never stored.
uint32_t a_box_rows(const GemmArgs& a, const GemmArgs* b) {
  const int64_t m = b ? std::max(a.M, b->M) : a.M;
  return m < BM ? (uint32_t)((m + 7) / 8 * 8) : (uint32_t)BM;
}

// Whether a launch needs the epilogue instance with the rarer features.
bool extra_args(const GemmArgs& a) {
  return a.epi.gate_scores || a.epi.sq_out || a.epi.cos_out || a.epi.nrm_psum || a.epi.out_f32;
}

template <int BN, bool DUAL, bool EXTRA>
cudaError_t launch_x(const GemmArgs& a, const GemmArgs* b, const Dev& dev) {
  using C = TileCfg<BN, DUAL>;
  if (a.a_gather || (b && b->a_gather)) return cudaErrorInvalidValue;
  static int attr_done[64] = {0};
  int device = 0;
  cudaGetDevice(&device);
  if (device < 64 && !attr_done[device]) {
    cudaError_t e = cudaFuncSetAttribute(gemm_tc_kernel<BN, DUAL, EXTRA>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM_BYTES);
    if (e != cudaSuccess) return e;
    attr_done[device] = 1;
  }
  CUtensorMap tm[4];
  GemmDev p, p2;
  cudaError_t e = prepare<DUAL>(a, b, a_box_rows(a, b), BN, BN, dev, tm, p, p2);
  if (e != cudaSuccess) return e;
  int64_t num_tiles = ((a.M + BM - 1) / BM) * ((a.N + p.bn - 1) / p.bn);
  if (b) num_tiles += ((b->M + BM - 1) / BM) * ((b->N + p2.bn - 1) / p2.bn);
  const int grid = (int)(num_tiles < dev.num_sms ? num_tiles : dev.num_sms);
  return launch_pdl(gemm_tc_kernel<BN, DUAL, EXTRA>, dim3(grid), dim3(kThreads), C::SMEM_BYTES,
                    dev.stream, tm[0], tm[1], tm[2], tm[3], p, p2);
}

template <int BN, bool DUAL>
cudaError_t launch(const GemmArgs& a, const GemmArgs* b, const Dev& dev) {
  return (extra_args(a) || (b && extra_args(*b))) ? launch_x<BN, DUAL, true>(a, b, dev)
                                                  : launch_x<BN, DUAL, false>(a, b, dev);
}

template <int BN, bool DUAL, bool EXTRA>
cudaError_t launch_pair_x(const GemmArgs& a, const GemmArgs* b, const Dev& dev) {
  using C = TileCfg<BN, DUAL, true>;
  static int attr_done[64] = {0};
  int device = 0;
  cudaGetDevice(&device);
  if (device < 64 && !attr_done[device]) {
    cudaError_t e = cudaFuncSetAttribute(gemm_tc2_kernel<BN, DUAL, EXTRA>,
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
    cudaError_t e = cudaOccupancyMaxActiveClusters(&n, gemm_tc2_kernel<BN, DUAL, EXTRA>, &cfg);
    if (e != cudaSuccess || n <= 0) return e != cudaSuccess ? e : cudaErrorInvalidConfiguration;
    max_pairs[device] = n;
  }
  const int64_t cap = device < 64 ? max_pairs[device] : dev.num_sms / 2;
  CUtensorMap tm[4];
  GemmDev p, p2;
  GemmArgs a_full = a;
  a_full.tile_n = 0;   // CTA pairs: full-width tiles only
  GemmArgs b_full;
  if (b) {
    b_full = *b;
    b_full.tile_n = 0;
  }
  cudaError_t e = prepare<DUAL>(a_full, b ? &b_full : nullptr, BM, BN, C::B_ROWS, dev, tm, p, p2);
  if (e != cudaSuccess) return e;
  int64_t num_tiles = ((a.M + 2 * BM - 1) / (2 * BM)) * ((a.N + BN - 1) / BN);
  if (b) num_tiles += ((b->M + 2 * BM - 1) / (2 * BM)) * ((b->N + BN - 1) / BN);
  const int64_t pairs = num_tiles < cap ? num_tiles : cap;
  return launch_pdl(gemm_tc2_kernel<BN, DUAL, EXTRA>, dim3((unsigned)(2 * pairs)), dim3(kThreads),
                    C::SMEM_BYTES, dev.stream, tm[0], tm[1], tm[2], tm[3], p, p2);
}

template <int BN, bool DUAL>
cudaError_t launch_pair(const GemmArgs& a, const GemmArgs* b, const Dev& dev) {
  return (extra_args(a) || (b && extra_args(*b))) ? launch_pair_x<BN, DUAL, true>(a, b, dev)
                                                  : launch_pair_x<BN, DUAL, false>(a, b, dev);
}

// Clusters of S CTAs of the split-K kernel that can be resident at once
// (cached per device and size; 0 if none).
template <int BN>
int sk_max_clusters(int S, const Dev& dev) {
  using C = TileCfg<BN, false>;
  static int cache[64][5] = {};
  static int attr_done[64] = {0};
  int device = 0;
  cudaGetDevice(&device);
  if (device >= 64 || S < 2 || S > 4) return 0;
  if (!attr_done[device]) {
    if (cudaFuncSetAttribute(gemm_tc_sk_kernel<BN, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             C::SMEM_BYTES) != cudaSuccess ||
        cudaFuncSetAttribute(gemm_tc_sk_kernel<BN, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             C::SMEM_BYTES) != cudaSuccess)
      return 0;
    attr_done[device] = 1;
  }
  if (!cache[device][S]) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(S * (dev.num_sms / S)));
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = C::SMEM_BYTES;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)S;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, gemm_tc_sk_kernel<BN, false>, &cfg) != cudaSuccess) n = 0;
    cache[device][S] = n > 0 ? n : -1;
  }
  return cache[device][S] > 0 ? cache[device][S] : 0;
}

// Tuning override: ADADSF_GEMM_SPLIT=1 disables the split-K kernel, 2 or 4
// forces that cluster size where it applies; unset or 0 chooses by the cost
// model.
int split_override() {
  static int v = -1;
  if (v < 0) {
    const char* e = getenv("ADADSF_GEMM_SPLIT");
    v = e ? atoi(e) : 0;
    if (v != 1 && v != 2 && v != 4) v = 0;
  }
  return v;
}

template <int BN>
cudaError_t launch_sk(const GemmArgs& a, const Dev& dev, int S) {
  using C = TileCfg<BN, false>;
  if (a.a_gather) return cudaErrorInvalidValue;
  CUtensorMap tm[4];
  GemmDev p, p2;
  GemmArgs a_full = a;
  a_full.tile_n = 0;
  cudaError_t e = prepare<false>(a_full, nullptr, a_box_rows(a, nullptr), BN, BN, dev, tm, p, p2);
  if (e != cudaSuccess) return e;
  const int64_t num_tiles = ((a.M + BM - 1) / BM) * ((a.N + BN - 1) / BN);
  if (extra_args(a))
    return launch_pdl_cluster(gemm_tc_sk_kernel<BN, true>, dim3((unsigned)(num_tiles * S)), dim3(kThreads),
                              C::SMEM_BYTES, dev.stream, S, tm[0], tm[1], tm[2], tm[3], p);
  return launch_pdl_cluster(gemm_tc_sk_kernel<BN, false>, dim3((unsigned)(num_tiles * S)), dim3(kThreads),
                            C::SMEM_BYTES, dev.stream, S, tm[0], tm[1], tm[2], tm[3], p);
}

// Plain and two-source projections (no SwiGLU, no router). Cost model in
// units of one k-block of one CTA: a tcgen05.mma with M = 128 takes about
// the same time for N = 128 as for N = 256, so a k-block costs the same for
// every tile width and a launch costs (tile rounds) x (k-blocks per CTA),
// plus its epilogue (per 32-column chunk of a thread) and, split along K,
// the exchange of partial tiles through the L2 (needs a.scratch). CTA pairs (256-row tiles) move half of the
// weight bytes per SM, the tie-breaker for large M.
cudaError_t gemm_plain(const GemmArgs& a, const Dev& dev) {
  // gathered A rows: CTA pairs (the only kernel that gathers)
  if (a.a_gather) return a.K2 > 0 ? cudaErrorInvalidValue : launch_pair<256, false>(a, nullptr, dev);
  const int num_kb = (a.K + (a.K2 > 0 ? a.K2 : 0) + BK - 1) / BK;
  const int64_t mb128 = (a.M + BM - 1) / BM, mb256 = (a.M + 2 * BM - 1) / (2 * BM);
  const int64_t t128 = mb128 * ((a.N + 127) / 128), t256 = mb128 * ((a.N + 255) / 256);
  const int64_t tpair = mb256 * ((a.N + 255) / 256);
  const int64_t sms = dev.num_sms;
  constexpr double kChunk = 2;      // 2 x (k-block cost) per epilogue chunk of 32 columns
  constexpr double kExchange = 4;   // partial-tile exchange through distributed shared memory
  // A k-block of a 256-column tile is the unit. With a single block of at most
  // 128 rows (a decode step's few rows) the product streams its weights and a
  // k-block costs in proportion to the weight rows it reads: narrower tiles,
  // on more CTAs, go faster.
  const bool stream_w = a.M <= BM;
  auto kb = [&](int bn) { return stream_w ? (double)num_kb * bn / 256.0 : (double)num_kb; };
  auto rounds = [](int64_t tiles, int64_t slots) { return (double)((tiles + slots - 1) / slots); };
  const double cost_pair = rounds(tpair, sms / 2) * num_kb + 4 * kChunk;
  const double cost256 = rounds(t256, sms) * kb(256) + 4 * kChunk;
  const double cost128 = rounds(t128, sms) * kb(128) + 2 * kChunk;
  double best = cost_pair;
  int pick = 0;   // 0 pair, 1 one-CTA 256, 2 one-CTA 128, 3 split 256, 4 split 128
  if (cost256 < best) { best = cost256; pick = 1; }
  if (cost128 < best) { best = cost128; pick = 2; }
  // Split along K (rotary tiles only with halves of at most 16 features,
  // which stay inside one 32-column chunk).
  const int force = split_override();
  int split_s = 0;
  const bool can_split = force != 1 && num_kb >= 2 && a.scratch != nullptr &&
                         (a.epi.rope_tab == nullptr || a.epi.rope_half <= 16);
  auto fits = [&](int64_t tiles, int S, int bn) {
    return (size_t)(tiles * S) * BM * bn * 4 <= a.scratch_bytes;
  };
  if (can_split) {
    for (int S = 2; S <= 4; S += 2) {
      if (S > num_kb || (force && force != S)) continue;
      const double k256 = std::ceil(kb(256) / S) + kExchange, k128 = std::ceil(kb(128) / S) + kExchange;
      if (fits(t256, S, 256) && t256 <= sk_max_clusters<256>(S, dev)) {
        const double c = k256 + kChunk * ((256 / S / 32 + 1) / 2);
        if (c < best || force) { best = c; pick = 3; split_s = S; }
      }
      if (fits(t128, S, 128) && t128 <= sk_max_clusters<128>(S, dev)) {
        const double c = k128 + kChunk * ((128 / S / 32 + 1) / 2);
        if (c < best || (force && pick != 3)) { best = c; pick = 4; split_s = S; }
      }
    }
  }
  switch (pick) {
    case 0: return launch_pair<256, false>(a, nullptr, dev);
    case 1: return launch<256, false>(a, nullptr, dev);
    case 2: return launch<128, false>(a, nullptr, dev);
    case 3: return launch_sk<256>(a, dev, split_s);
    default: return launch_sk<128>(a, dev, split_s);
  }
}

}  // namespace

// Room for the partial tiles of up to 160 CTAs of 128 x 256 fp32 (every
// split the cost model can choose on a GPU with up to 160 SMs).
size_t gemm_split_scratch_bytes() { return (size_t)160 * BM * 256 * 4; }

cudaError_t gemm_bf16(const GemmArgs& a, const Dev& dev) {
  if (a.M <= 0) return cudaSuccess;
  if (a.a_gather && (a.epi.act == ACT_SWIGLU || a.a_gather_rows <= 0)) return cudaErrorInvalidValue;
  // SwiGLU: 256 x 128 gate/up tiles on CTA pairs when that still gives every
  // pair of SMs at least two tiles.
  if (a.epi.act == ACT_SWIGLU) {
    if (a.K2 > 0) return cudaErrorInvalidValue;
    const int64_t pair_tiles = ((a.M + 255) / 256) * ((a.N + 127) / 128);
    if (a.N % 128 == 0 && pair_tiles >= dev.num_sms) return launch_pair<128, true>(a, nullptr, dev);
    return launch<128, true>(a, nullptr, dev);
  }
  return gemm_plain(a, dev);
}

cudaError_t gemm_bf16_grouped(const GemmArgs& a, const GemmArgs& b, const Dev& dev) {
  if (a.a_gather || b.a_gather) return cudaErrorInvalidValue;
  if (a.M <= 0 && b.M <= 0) return cudaSuccess;
  if (a.M <= 0) return gemm_bf16(b, dev);
  if (b.M <= 0) return gemm_bf16(a, dev);
  auto plain = [](const GemmArgs& g) {
    return g.epi.act != ACT_SWIGLU && g.K2 == 0;
  };
  if (!plain(a) || !plain(b)) return cudaErrorInvalidValue;
  // Fewest rounds of tiles (a k-block costs the same for any tile width);
  // ties go to CTA pairs (half the weight bytes per SM), then to 256-wide
  // tiles. Problem `a` comes first in the tile order: pass the one with the
  // costlier epilogue as `a` so that it runs in the first round.
  // Cost in k-block units: rounds of tiles x k-blocks, plus the epilogue of
  // a last-round tile (per 32-column chunk of a thread: ~1.5 units, ~3 with
  // GELU). Giving the first problem half-width (128-column) tiles doubles
  // its tiles but halves their epilogue.
  auto tiles = [](const GemmArgs& g, int bm, int bn) { return ((g.M + bm - 1) / bm) * ((g.N + bn - 1) / bn); };
  auto chunk = [](const GemmArgs& g) -> int64_t { return g.epi.act == ACT_GELU ? 3 : 2; };
  const int64_t sms = dev.num_sms;
  const int64_t kb = (std::max(a.K, b.K) + BK - 1) / BK;
  const int64_t epi_w = 4 * std::max(chunk(a), chunk(b));
  const int64_t c_pair = (tiles(a, 256, 256) + tiles(b, 256, 256) + sms / 2 - 1) / (sms / 2) * kb + epi_w;
  const int64_t c256 = (tiles(a, 128, 256) + tiles(b, 128, 256) + sms - 1) / sms * kb + epi_w;
  const int64_t c_half = (tiles(a, 128, 128) + tiles(b, 128, 256) + sms - 1) / sms * kb +
                         std::max(2 * chunk(a), 4 * chunk(b));
  const int64_t c128 = (tiles(a, 128, 128) + tiles(b, 128, 128) + sms - 1) / sms * kb +
                       2 * std::max(chunk(a), chunk(b));
  const int64_t best = std::min(std::min(c_pair, c256), std::min(c_half, c128));
  if (c_pair == best) return launch_pair<256, false>(a, &b, dev);
  if (c256 == best) return launch<256, false>(a, &b, dev);
  if (c_half == best) {
    GemmArgs a_half = a;
    a_half.tile_n = 128;
    return launch<256, false>(a_half, &b, dev);
  }
  return launch<128, false>(a, &b, dev);
}

}  // namespace adadsf
