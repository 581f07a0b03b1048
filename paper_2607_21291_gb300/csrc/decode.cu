// Autoregressive decode with a cache of kept tokens only. The paper (Sec.
// 3.4) defines the sparse forward over a whole sequence and is silent on
// generation; the reading implemented here: a generated token is kept at
// layer l when its router score beats the lowest score the layer kept in the
// prompt (the K-th largest of the Top-K, +inf when the layer kept nothing);
// a kept token attends to the layer's cached kept tokens and itself (rotary
// at original positions), gets the layer's residual delta, and its key and
// value join the cache; a skipped token bypasses the layer.
//
// Cache (one caller buffer, all device memory):
//   header   {T_cur, C_max, L, B} int32, padded to 256 bytes
//   lens     [L][B] int32     kept tokens cached per layer and sequence
//   thr      [L][B] fp32      keep thresholds
//   rope     [C_max][rot/2]   (cos, sin) fp32 pairs of every position
//   K, V     [L][B][Hkv][C_max][head_dim] each, storage dtype
// Every kernel reads positions and lengths from the cache, so a decode step
// has fixed launch arguments (capturable once in a CUDA graph).
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace adadsf {
namespace {

constexpr int kDecThreads = 128;        // 4 warps per fp32 attention CTA
constexpr int kMaxGroup = 16;           // query heads per key/value head
constexpr int kDecTK = 64;              // keys per tile (split granularity, ring stage)
constexpr int kDecStages = 3;           // ring stages of the bf16 kernel
constexpr int kDecWarps = 4;            // consumer warps of the bf16 kernel, 16 keys of a tile each
constexpr int kDecTcThreads = 32 * (kDecWarps + 1);
constexpr int kRopeThreads = 1024;       // rotary + cache append: threads per sequence

// ---------------------------------------------------------------- prefill -> cache
// K and V of the kept (packed) rows m = b K + j of one layer into the cache:
// row j of sequence b, every key/value head.
template <typename T>
__global__ void kv_fill_kernel(const T* qkv, int64_t ld, int q, int kvw, int B, int K, int hd,
                               int C_max, T* kc, T* vc) {
  pdl_trigger();
  pdl_wait();
  constexpr int V = Elem<T>::kVec;
  const int nvec = kvw / V;                       // 16-byte vectors of one row's keys
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (int64_t)B * K * nvec) return;
  const int64_t m = i / nvec;
  const int c = (int)(i % nvec) * V;              // feature within the kv width
  const int b = (int)(m / K), j = (int)(m % K);
  const int h = c / hd, e = c % hd;
  const int64_t dst = (((int64_t)b * (kvw / hd) + h) * C_max + j) * hd + e;
  *reinterpret_cast<uint4*>(kc + dst) = *reinterpret_cast<const uint4*>(qkv + m * ld + q + c);
  *reinterpret_cast<uint4*>(vc + dst) = *reinterpret_cast<const uint4*>(qkv + m * ld + q + kvw + c);
}

// Per sequence b: lens[b] = K and thr[b] = the lowest router score among its
// kept positions (+inf when K = 0). One block per sequence.
__global__ void kv_threshold_kernel(const float* scores, const int32_t* idx, int T, int K,
                                    int32_t* lens, float* thr) {
  pdl_trigger();
  pdl_wait();
  __shared__ float red[32];
  __shared__ int any_nan;
  const int b = blockIdx.x;
  if (threadIdx.x == 0) any_nan = 0;
  __syncthreads();
  float m = INFINITY;
  for (int j = threadIdx.x; j < K; j += blockDim.x) {
    const float s = scores[(int64_t)b * T + idx[(int64_t)b * K + j]];
    if (isnan(s)) any_nan = 1;   // a NaN was kept (fewer numbers than K): it is the minimum
    m = fminf(m, s);
  }
  for (int o = 16; o > 0; o >>= 1) m = fminf(m, __shfl_xor_sync(0xffffffffu, m, o));
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = m;
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int w = 1; w < (int)(blockDim.x >> 5); ++w) m = fminf(m, red[w]);
    lens[b] = K;
    thr[b] = any_nan ? NAN : m;
  }
}

__global__ void cache_header_kernel(int32_t* hdr, int T, int C_max, int L, int B) {
  pdl_trigger();
  pdl_wait();
  if (threadIdx.x == 0) {
    hdr[0] = T;
    hdr[1] = C_max;
    hdr[2] = L;
    hdr[3] = B;
  }
}

// ---------------------------------------------------------------- decode step
// Keep decision of the new token of every sequence at one layer, its
// position, and the packed-row map of the projections (rows[b] = b if kept,
// -1 if it bypasses the layer: the residual scatter then skips it). A tie
// loses and NaN never wins. A cache not filled by a prefill of this shape, or
// no room left in its rotary table, raises DEVERR_INDEX and the position is
// clamped into range. (The same rule runs inside decide_norm_kernel when the
// router is not forked onto a stream of its own.)
__global__ void decode_decide_kernel(const float* scores, const float* thr, const int32_t* hdr, int B,
                                     int C_max, int32_t* rows, int32_t* pos, int32_t* kept_out, int* err) {
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  int t = hdr[0];
  if (hdr[1] != C_max || t < 0 || t >= C_max) {
    set_device_error(err, DEVERR_INDEX);
    t = t < 0 ? 0 : (t >= C_max ? C_max - 1 : t);
  }
  const bool keep = scores[b] > thr[b];
  rows[b] = keep ? b : -1;
  pos[b] = t;
  if (kept_out) kept_out[b] = keep ? 1 : 0;
}

// Attention of the new token of sequence b, query heads h G .. h G + G - 1
// (G = Hq / Hkv) of key/value head h, over split s of the n = lens[b] cached
// keys (the token's own key is already appended). The splits cover [0, n) in
// whole tiles of kDecTK keys; a split's partial (row max in log2 units, sum,
// unnormalised output) per query head goes to part_ml / part_o for the
// combine step. Scores carry log2(e) / sqrt(hd), so the softmax runs on exp2.
__device__ __forceinline__ void dec_split_range(int n, int nsplit, int s, int& lo, int& hi) {
  const int per = ((n + nsplit - 1) / nsplit + kDecTK - 1) / kDecTK * kDecTK;
  lo = min(n, s * per);
  hi = min(n, lo + per);
}

// fp32 storage: CUDA cores, each warp of the CTA takes every 4th key with an
// online softmax per query head.
__global__ void __launch_bounds__(kDecThreads)
    decode_attn_f32_kernel(const float* qkv, int64_t ld, int Hq, int Hkv, int hd, const float* kc,
                           const float* vc, const int32_t* lens, int C_max, int nsplit, float scale_log2,
                           float* part_o, float2* part_ml) {
  pdl_trigger();
  pdl_wait();
  const int s = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int G = Hq / Hkv;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int per = hd / 32;                        // features per lane (2 or 4)
  int n = lens[b];
  n = n < 0 ? 0 : (n > C_max ? C_max : n);
  int lo, hi;
  dec_split_range(n, nsplit, s, lo, hi);
  const float* qrow = qkv + (int64_t)b * ld;
  float qv[kMaxGroup][4];
  for (int g = 0; g < G; ++g)
    for (int i = 0; i < per; ++i) qv[g][i] = qrow[(h * G + g) * hd + lane * per + i] * scale_log2;
  float mx[kMaxGroup], sm[kMaxGroup], acc[kMaxGroup][4];
  for (int g = 0; g < G; ++g) {
    mx[g] = -INFINITY;
    sm[g] = 0.f;
    for (int i = 0; i < per; ++i) acc[g][i] = 0.f;
  }
  const int64_t base = ((int64_t)b * Hkv + h) * C_max;
  for (int j = lo + warp; j < hi; j += 4) {
    const float* kr = kc + (base + j) * hd;
    const float* vr = vc + (base + j) * hd;
    float kf[4], vf[4];
    for (int i = 0; i < per; ++i) {
      kf[i] = kr[lane * per + i];
      vf[i] = vr[lane * per + i];
    }
    for (int g = 0; g < G; ++g) {
      float dot = 0.f;
      for (int i = 0; i < per; ++i) dot = fmaf(qv[g][i], kf[i], dot);
      dot = warp_sum(dot);
      const float mnew = fmaxf(mx[g], dot);
      const float corr = exp2f(mx[g] - mnew);
      const float pj = exp2f(dot - mnew);
      sm[g] = sm[g] * corr + pj;
      for (int i = 0; i < per; ++i) acc[g][i] = fmaf(acc[g][i], corr, pj * vf[i]);
      mx[g] = mnew;
    }
  }
  // merge the 4 warps' partials per head in shared memory
  __shared__ float s_ml[4][kMaxGroup][2];
  __shared__ float s_o[4][kMaxGroup][128];
  for (int g = 0; g < G; ++g) {
    if (lane == 0) {
      s_ml[warp][g][0] = mx[g];
      s_ml[warp][g][1] = sm[g];
    }
    for (int i = 0; i < per; ++i) s_o[warp][g][lane * per + i] = acc[g][i];
  }
  __syncthreads();
  for (int k = threadIdx.x; k < G * hd; k += kDecThreads) {
    const int g = k / hd, e = k % hd;
    float m = -INFINITY;
    for (int w = 0; w < 4; ++w) m = fmaxf(m, s_ml[w][g][0]);
    float l = 0.f, o = 0.f;
    if (m > -INFINITY) {
      for (int w = 0; w < 4; ++w) {
        const float c = exp2f(s_ml[w][g][0] - m);
        l += s_ml[w][g][1] * c;
        o += s_o[w][g][e] * c;
      }
    }
    const int64_t slot = ((int64_t)b * Hq + h * G + g) * nsplit + s;
    part_o[slot * hd + e] = o;
    if (e == 0) part_ml[slot] = make_float2(m, l);
  }
}

// bf16 storage: tensor cores (warp-level mma.sync m16n8k16, bf16 in, fp32
// accumulate). The G query heads of the group are the 16 rows of the A
// operand (rows >= G are zero), so one key tile costs the same whatever G.
// Warp 4 streams the key/value tiles of the split through a ring of
// kDecStages stages with 2-D TMA copies (128-byte swizzle, 64 features per
// box); warps 0..3 each take 16 keys of a tile:
//   S (16 x 16)  = Q (16 x HD) . K^T           (ldmatrix from the swizzled tile)
//   online softmax per row (exp2; the 4 lanes of a quad share a row)
//   O (16 x HD) += P (16 x 16, bf16) . V (16 x HD)   (ldmatrix.trans)
// and the four warps' (max, sum, O) merge in shared memory at the end.
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t (&r)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t (&r)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
// D += A . B for one m16n8k16 tile (A row-major 16 x 16, B column-major 16 x 8).
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                               uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
// Byte offset of (row, col) in a ring tile: boxes of 64 features (128 bytes)
// side by side, each kDecTK rows of 128 bytes with the 16-byte chunks of a
// row permuted by XOR with (row mod 8), as the TMA 128-byte swizzle writes them.
__device__ __forceinline__ uint32_t dec_swz(int row, int col) {
  return (uint32_t)((col >> 6) * (kDecTK * 128) + row * 128 + ((((col & 63) >> 3) ^ (row & 7)) << 4));
}
__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xffff0000u); }

template <int HD>
struct DecTc {
  static constexpr int TILE = HD / 64 * kDecTK * 128;     // K (or V) of one stage, bytes
  static constexpr int STAGE = 2 * TILE;
  static constexpr int RING = kDecStages * STAGE;
  static constexpr int OLD = HD + 8;                      // merge row stride (floats), padded
  static constexpr int MERGE = kDecWarps * 16 * (OLD + 2) * 4;
  static_assert(MERGE <= RING, "the merge area reuses the ring");
  static constexpr int SMEM = RING + 1024;                // + alignment slack
};

template <int HD>
__global__ void __launch_bounds__(kDecTcThreads)
    decode_attn_tc_kernel(const __grid_constant__ CUtensorMap tk, const __grid_constant__ CUtensorMap tv,
                          const bf16* qkv, int64_t ld, int Hq, int Hkv, const int32_t* lens, int C_max,
                          int nsplit, float scale_log2, float* part_o, float2* part_ml, int* err,
                          unsigned long long timeout_ns) {
  using C = DecTc<HD>;
  extern __shared__ __align__(1024) uint8_t dsm[];
  __shared__ __align__(8) uint64_t bars[2 * kDecStages];
  __shared__ int abort_s;
  const uint32_t ring = (smem_u32(dsm) + 1023u) & ~1023u;
  uint8_t* ring_p = dsm + (ring - smem_u32(dsm));
  const uint32_t full0 = smem_u32(&bars[0]), empty0 = smem_u32(&bars[kDecStages]);
  volatile int* abort_flag = &abort_s;
  const int s = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int G = Hq / Hkv;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int i = 0; i < kDecStages; ++i) {
      mbar_init(full0 + 8 * i, 1);
      mbar_init(empty0 + 8 * i, kDecWarps);
    }
    abort_s = 0;
    fence_barrier_init();
  }
  if (warp == kDecWarps && lane == 0) {
    tma_prefetch_desc(&tk);
    tma_prefetch_desc(&tv);
  }
  __syncthreads();
  pdl_trigger();
  pdl_wait();
  int n = lens[b];
  n = n < 0 ? 0 : (n > C_max ? C_max : n);
  int lo, hi;
  dec_split_range(n, nsplit, s, lo, hi);
  const int ntiles = (hi - lo + kDecTK - 1) / kDecTK;
  const int row0 = (b * Hkv + h) * C_max + lo;            // first key's row in the layer's cache

  const int gid = lane >> 2, tig = lane & 3;
  float o[HD / 8][4];
  float m_r[2] = {-INFINITY, -INFINITY}, l_r[2] = {0.f, 0.f};   // rows gid, gid + 8
#pragma unroll
  for (int i = 0; i < HD / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;

  if (warp == kDecWarps) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      int t = 0;
      for (; t < ntiles; ++t) {
        const int st = t % kDecStages;
        if (!mbar_wait_bounded(empty0 + 8 * st, ((t / kDecStages) & 1) ^ 1, abort_flag, err, timeout_ns)) break;
        const uint32_t fb = full0 + 8 * st;
        mbar_arrive_expect_tx(fb, C::STAGE);
        const uint32_t dk = ring + st * C::STAGE;
#pragma unroll
        for (int x = 0; x < HD / 64; ++x) {
          tma_load_2d(dk + x * kDecTK * 128, &tk, x * 64, row0 + t * kDecTK, fb);
          tma_load_2d(dk + C::TILE + x * kDecTK * 128, &tv, x * 64, row0 + t * kDecTK, fb);
        }
      }
      // drain: the copies issued last into each stage have landed
      for (int st = 0; st < kDecStages && st < t; ++st) {
        const int last = st + ((t - 1 - st) / kDecStages) * kDecStages;
        mbar_wait_drain(full0 + 8 * st, (uint32_t)((last / kDecStages) & 1), timeout_ns);
      }
    }
  } else {
    // ------------------------------------------------------------ consumers
    // Q of the group as A fragments (rows g >= G zero), once
    uint32_t qa[HD / 16][4];
    const bf16* qrow = qkv + (int64_t)b * ld + (int64_t)h * G * HD;
    const bool r0 = gid < G, r1 = gid + 8 < G;
#pragma unroll
    for (int ks = 0; ks < HD / 16; ++ks) {
      const int c = ks * 16 + tig * 2;
      qa[ks][0] = r0 ? *reinterpret_cast<const uint32_t*>(qrow + gid * HD + c) : 0u;
      qa[ks][1] = r1 ? *reinterpret_cast<const uint32_t*>(qrow + (gid + 8) * HD + c) : 0u;
      qa[ks][2] = r0 ? *reinterpret_cast<const uint32_t*>(qrow + gid * HD + c + 8) : 0u;
      qa[ks][3] = r1 ? *reinterpret_cast<const uint32_t*>(qrow + (gid + 8) * HD + c + 8) : 0u;
    }
    const int mi = lane >> 3, mr = lane & 7;   // ldmatrix: this lane's matrix and row
    for (int t = 0; t < ntiles; ++t) {
      const int st = t % kDecStages;
      const bool ok = mbar_wait_bounded(full0 + 8 * st, (t / kDecStages) & 1, abort_flag, err, timeout_ns);
      if (!__all_sync(0xffffffffu, ok)) break;
      const uint32_t kt = ring + st * C::STAGE, vt = kt + C::TILE;
      const int kw = warp * 16;                             // this warp's keys within the tile
      float sc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
#pragma unroll
      for (int ks = 0; ks < HD / 16; ++ks) {
        uint32_t kb[4];
        ldsm_x4(kt + dec_swz(kw + (mi >> 1) * 8 + mr, ks * 16 + (mi & 1) * 8), kb);
        mma_bf16_16816(sc[0], qa[ks], kb[0], kb[1]);
        mma_bf16_16816(sc[1], qa[ks], kb[2], kb[3]);
      }
      // online softmax over the warp's 16 keys; key j0 + 8 nt + 2 tig + e
      const int j0 = lo + t * kDecTK + kw;
      float tmax[2] = {-INFINITY, -INFINITY};
#pragma unroll
      for (int nt = 0; nt < 2; ++nt)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const bool valid = j0 + nt * 8 + tig * 2 + (e & 1) < hi;
          sc[nt][e] = valid ? sc[nt][e] * scale_log2 : -INFINITY;
          tmax[e >> 1] = fmaxf(tmax[e >> 1], sc[nt][e]);
        }
      float corr[2], base[2];
#pragma unroll
      for (int r = 0; r < 2; ++r) {
        tmax[r] = fmaxf(tmax[r], __shfl_xor_sync(0xffffffffu, tmax[r], 1));
        tmax[r] = fmaxf(tmax[r], __shfl_xor_sync(0xffffffffu, tmax[r], 2));
        const float mn = fmaxf(m_r[r], tmax[r]);
        base[r] = mn == -INFINITY ? 0.f : mn;
        corr[r] = exp2f(m_r[r] - base[r]);
        m_r[r] = mn;
      }
      uint32_t pa[4];
      float psum[2] = {0.f, 0.f};
#pragma unroll
      for (int nt = 0; nt < 2; ++nt)
#pragma unroll
        for (int r = 0; r < 2; ++r) {
          const uint32_t pk = pack_bf16x2(exp2f(sc[nt][2 * r] - base[r]), exp2f(sc[nt][2 * r + 1] - base[r]));
          pa[nt * 2 + r] = pk;
          psum[r] += bf16_lo(pk) + bf16_hi(pk);
        }
#pragma unroll
      for (int r = 0; r < 2; ++r) l_r[r] = l_r[r] * corr[r] + psum[r];
#pragma unroll
      for (int i = 0; i < HD / 8; ++i) {
        o[i][0] *= corr[0];
        o[i][1] *= corr[0];
        o[i][2] *= corr[1];
        o[i][3] *= corr[1];
      }
#pragma unroll
      for (int np = 0; np < HD / 16; ++np) {
        uint32_t vb[4];
        ldsm_x4_t(vt + dec_swz(kw + (mi & 1) * 8 + mr, np * 16 + (mi >> 1) * 8), vb);
        mma_bf16_16816(o[2 * np], pa, vb[0], vb[1]);
        mma_bf16_16816(o[2 * np + 1], pa, vb[2], vb[3]);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(empty0 + 8 * st);
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      l_r[r] += __shfl_xor_sync(0xffffffffu, l_r[r], 1);
      l_r[r] += __shfl_xor_sync(0xffffffffu, l_r[r], 2);
    }
  }
  __syncthreads();   // the ring is drained and read: its memory takes the merge
  float* mo = reinterpret_cast<float*>(ring_p);                     // [warp][16][OLD]
  float* mml = mo + kDecWarps * 16 * C::OLD;                        // [warp][16][2]
  if (warp < kDecWarps) {
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const int row = gid + 8 * r;
      if (row < G) {
        float* dst = mo + (warp * 16 + row) * C::OLD + tig * 2;
#pragma unroll
        for (int i = 0; i < HD / 8; ++i) *reinterpret_cast<float2*>(dst + i * 8) = make_float2(o[i][2 * r], o[i][2 * r + 1]);
        if (tig == 0) {
          mml[(warp * 16 + row) * 2] = m_r[r];
          mml[(warp * 16 + row) * 2 + 1] = l_r[r];
        }
      }
    }
  }
  __syncthreads();
  for (int k = threadIdx.x; k < G * HD; k += kDecTcThreads) {
    const int g = k / HD, e = k % HD;
    float m = -INFINITY;
#pragma unroll
    for (int w = 0; w < kDecWarps; ++w) m = fmaxf(m, mml[(w * 16 + g) * 2]);
    float l = 0.f, ov = 0.f;
    if (m > -INFINITY) {
#pragma unroll
      for (int w = 0; w < kDecWarps; ++w) {
        const float c = exp2f(mml[(w * 16 + g) * 2] - m);
        l += mml[(w * 16 + g) * 2 + 1] * c;
        ov += mo[(w * 16 + g) * C::OLD + e] * c;
      }
    }
    const int64_t slot = ((int64_t)b * Hq + h * G + g) * nsplit + s;
    part_o[slot * HD + e] = ov;
    if (e == 0) part_ml[slot] = make_float2(m, l);
  }
}

// out[b][head] = sum_s 2^(m_s - m) o_s / sum_s 2^(m_s - m) l_s over the
// splits; a head with no key at all (an empty cache) gets zeros.
template <typename T>
__global__ void decode_combine_kernel(const float* part_o, const float2* part_ml, int Hq, int hd,
                                      int nsplit, T* out, int64_t ld_out) {
  pdl_trigger();
  pdl_wait();
  const int hq = blockIdx.x, b = blockIdx.y;
  const int64_t slot0 = ((int64_t)b * Hq + hq) * nsplit;
  float m = -INFINITY;
  for (int s = 0; s < nsplit; ++s) m = fmaxf(m, part_ml[slot0 + s].x);
  for (int e = threadIdx.x; e < hd; e += blockDim.x) {
    float l = 0.f, o = 0.f;
    for (int s = 0; s < nsplit; ++s) {
      const float2 ml = part_ml[slot0 + s];
      if (ml.x == -INFINITY) continue;
      const float c = exp2f(ml.x - m);
      l += ml.y * c;
      o += part_o[(slot0 + s) * hd + e] * c;
    }
    out[(int64_t)b * ld_out + hq * hd + e] = Elem<T>::from_f(l > 0.f ? o / l : 0.f);
  }
}

// Rotary embedding of the new tokens' query and key heads at their positions
// (feature i < half pairs with i + half, as in the prefill), fused with the
// cache append: a kept token's rotated key and its value join the layer's
// cache at lens[b], then lens[b] += 1. One block per sequence b, wide enough
// that each thread has one or two pairs (the launch is latency bound).
template <typename T>
__global__ void __launch_bounds__(kRopeThreads) rope_append_kernel(T* qkv, int64_t ld, int Hq, int Hkv, int hd, int half,
                                   const int32_t* pos, const float2* tab, const int32_t* rows,
                                   int32_t* lens, int C_max, T* kc, T* vc, int* err) {
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x;
  T* row = qkv + (int64_t)b * ld;
  const int q = Hq * hd, kvw = Hkv * hd;
  bool append = rows[b] >= 0;
  const int len = lens[b];
  if (append && (len < 0 || len >= C_max)) {
    if (threadIdx.x == 0) set_device_error(err, DEVERR_INDEX);
    append = false;
  }
  const float2* tab_row = tab + (int64_t)pos[b] * half;
  // rotated pairs of every query and key head
  for (int k = threadIdx.x; k < (Hq + Hkv) * half; k += blockDim.x) {
    const int h = k / half, i = k % half;
    T* base = row + (int64_t)h * hd;
    const float2 cs = tab_row[i];
    const float a = Elem<T>::to_f(base[i]);
    const float c = Elem<T>::to_f(base[i + half]);
    const T ra = Elem<T>::from_f(a * cs.x - c * cs.y);
    const T rc = Elem<T>::from_f(c * cs.x + a * cs.y);
    base[i] = ra;
    base[i + half] = rc;
    if (append && h >= Hq) {
      const int64_t dst = (((int64_t)b * Hkv + (h - Hq)) * C_max + len) * hd;
      kc[dst + i] = ra;
      kc[dst + i + half] = rc;
    }
  }
  if (append) {
    // key features past the rotary pairs, and the values
    for (int c = threadIdx.x; c < kvw; c += blockDim.x) {
      const int h = c / hd, e = c % hd;
      const int64_t dst = (((int64_t)b * Hkv + h) * C_max + len) * hd + e;
      if (e >= 2 * half) kc[dst] = row[q + c];
      vc[dst] = row[q + kvw + c];
    }
  }
  __syncthreads();
  if (threadIdx.x == 0 && append) lens[b] = len + 1;
}

__global__ void decode_advance_kernel(int32_t* hdr) {
  pdl_trigger();
  pdl_wait();
  if (threadIdx.x == 0) hdr[0] += 1;
}

}  // namespace

// ---------------------------------------------------------------- host side
int decode_splits(int B, int Hkv, int C_max, int num_sms) {
  // two CTAs of the bf16 kernel per SM in one wave, at least one tile a split
  int s = 2 * num_sms / (B * Hkv);
  const int max_s = (C_max + kDecTK - 1) / kDecTK;
  if (s > max_s) s = max_s;
  if (s > 64) s = 64;
  return s < 1 ? 1 : s;
}

cudaError_t kv_fill(int dtype, const void* qkv, int64_t ld, int q, int kvw, int B, int K, int hd,
                    int C_max, void* kc, void* vc, const Dev& dev) {
  const int V = dtype == kBF16 ? 8 : 4;
  const int64_t n = (int64_t)B * K * (kvw / V);
  if (n <= 0) return cudaSuccess;
  const dim3 grid((unsigned)((n + 255) / 256));
  if (dtype == kBF16)
    return launch_pdl(kv_fill_kernel<bf16>, grid, dim3(256), 0, dev.stream, static_cast<const bf16*>(qkv), ld,
                      q, kvw, B, K, hd, C_max, static_cast<bf16*>(kc), static_cast<bf16*>(vc));
  return launch_pdl(kv_fill_kernel<float>, grid, dim3(256), 0, dev.stream, static_cast<const float*>(qkv), ld,
                    q, kvw, B, K, hd, C_max, static_cast<float*>(kc), static_cast<float*>(vc));
}

cudaError_t kv_threshold(const float* scores, const int32_t* idx, int B, int T, int K, int32_t* lens,
                         float* thr, const Dev& dev) {
  if (B <= 0) return cudaSuccess;
  return launch_pdl(kv_threshold_kernel, dim3(B), dim3(256), 0, dev.stream, scores, idx, T, K, lens, thr);
}

cudaError_t cache_header(int32_t* hdr, int T, int C_max, int L, int B, const Dev& dev) {
  return launch_pdl(cache_header_kernel, dim3(1), dim3(32), 0, dev.stream, hdr, T, C_max, L, B);
}

template <int HD>
static cudaError_t launch_decode_tc(const CUtensorMap& tk, const CUtensorMap& tv, const bf16* qkv, int64_t ld,
                                    int Hq, int Hkv, const int32_t* lens, int C_max, int B, int ns,
                                    float scale_log2, float* part_o, float2* part_ml, const Dev& dev) {
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(decode_attn_tc_kernel<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         DecTc<HD>::SMEM);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  return launch_pdl(decode_attn_tc_kernel<HD>, dim3(ns, Hkv, B), dim3(kDecTcThreads), (size_t)DecTc<HD>::SMEM,
                    dev.stream, tk, tv, qkv, ld, Hq, Hkv, lens, C_max, ns, scale_log2, part_o, part_ml, dev.err,
                    kWaitTimeoutNs);
}

cudaError_t decode_decide(const float* scores, const float* thr, const int32_t* hdr, int B, int C_max,
                          int32_t* rows, int32_t* pos, int32_t* kept_out, const Dev& dev) {
  return launch_pdl(decode_decide_kernel, dim3((B + 127) / 128), dim3(128), 0, dev.stream, scores, thr, hdr, B,
                    C_max, rows, pos, kept_out, dev.err);
}

cudaError_t decode_attention(int dtype, const void* qkv, int64_t ld, int Hq, int Hkv, int hd, const void* kc,
                             const void* vc, const int32_t* lens, int C_max, int B, float* part_o,
                             float2* part_ml, void* out, int64_t ld_out, const Dev& dev) {
  if (B <= 0) return cudaSuccess;
  if (Hq % Hkv != 0 || Hq / Hkv > kMaxGroup || (hd != 64 && hd != 128)) return cudaErrorInvalidValue;
  const int ns = decode_splits(B, Hkv, C_max, dev.num_sms);
  if ((int64_t)ns * (C_max + kDecTK) > INT32_MAX) return cudaErrorInvalidValue;   // split bounds stay in int
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)hd);   // log2(e) / sqrt(hd)
  cudaError_t e;
  if (dtype == kBF16) {
    // the layer's keys (values) as one [B Hkv C_max, hd] matrix; a tile's
    // first row must fit the copy's 32-bit coordinate
    const int64_t rows = (int64_t)B * Hkv * C_max;
    if (rows + kDecTK > INT32_MAX) return cudaErrorInvalidValue;
    CUtensorMap tk, tv;
    if (!make_tmap_bf16(&tk, kc, (uint64_t)rows, (uint64_t)hd, (uint64_t)hd, 64, kDecTK) ||
        !make_tmap_bf16(&tv, vc, (uint64_t)rows, (uint64_t)hd, (uint64_t)hd, 64, kDecTK))
      return cudaErrorInvalidValue;
    const bf16* q = static_cast<const bf16*>(qkv);
    e = hd == 128 ? launch_decode_tc<128>(tk, tv, q, ld, Hq, Hkv, lens, C_max, B, ns, scale_log2, part_o, part_ml, dev)
                  : launch_decode_tc<64>(tk, tv, q, ld, Hq, Hkv, lens, C_max, B, ns, scale_log2, part_o, part_ml, dev);
  } else {
    e = launch_pdl(decode_attn_f32_kernel, dim3(ns, Hkv, B), dim3(kDecThreads), 0, dev.stream,
                   static_cast<const float*>(qkv), ld, Hq, Hkv, hd, static_cast<const float*>(kc),
                   static_cast<const float*>(vc), lens, C_max, ns, scale_log2, part_o, part_ml);
  }
  if (e != cudaSuccess) return e;
  if (dtype == kBF16)
    return launch_pdl(decode_combine_kernel<bf16>, dim3(Hq, B), dim3(128), 0, dev.stream, part_o, part_ml, Hq,
                      hd, ns, static_cast<bf16*>(out), ld_out);
  return launch_pdl(decode_combine_kernel<float>, dim3(Hq, B), dim3(128), 0, dev.stream, part_o, part_ml, Hq, hd,
                    ns, static_cast<float*>(out), ld_out);
}

cudaError_t rope_append(int dtype, void* qkv, int64_t ld, int Hq, int Hkv, int hd, int rotary_dim, int B,
                        const int32_t* rows, const int32_t* pos, const float2* tab, int32_t* lens, int C_max,
                        void* kc, void* vc, const Dev& dev) {
  if (B <= 0) return cudaSuccess;
  const int half = rotary_dim / 2;
  if (dtype == kBF16)
    return launch_pdl(rope_append_kernel<bf16>, dim3(B), dim3(kRopeThreads), 0, dev.stream, static_cast<bf16*>(qkv), ld, Hq,
                      Hkv, hd, half, pos, tab, rows, lens, C_max, static_cast<bf16*>(kc), static_cast<bf16*>(vc),
                      dev.err);
  return launch_pdl(rope_append_kernel<float>, dim3(B), dim3(kRopeThreads), 0, dev.stream, static_cast<float*>(qkv), ld, Hq,
                    Hkv, hd, half, pos, tab, rows, lens, C_max, static_cast<float*>(kc), static_cast<float*>(vc),
                    dev.err);
}

cudaError_t decode_advance(int32_t* hdr, const Dev& dev) {
  return launch_pdl(decode_advance_kernel, dim3(1), dim3(32), 0, dev.stream, hdr);
}

}  // namespace adadsf
