// Row-wise kernels of the depth-sparse layer: embedding, fused gather + norm,
// rotary embedding at original positions, fp32 router, per-sequence Top-K,
// the Eq. 4 similarity reduction, and the bounded-wait self-test.
// All are HBM-bound: rows are moved as 16-byte vectors, one warp per row.
#include <algorithm>
#include <mutex>
#include <type_traits>

#include "common.cuh"
#include "internal.h"
#include "topk.cuh"

namespace adadsf {
namespace {

constexpr int kMaxChunks = 16;  // per-lane 16-byte vectors held in registers (d <= 16*32*vec)

// ---------------------------------------------------------------- embedding
template <typename T>
__global__ void embed_kernel(const int32_t* ids, int64_t n, const T* table, int vocab, int d,
                             T* out, int* err) {
  pdl_trigger();
  pdl_wait();
  constexpr int V = Elem<T>::kVec;
  const int64_t row = (int64_t)blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
  const int lane = threadIdx.x & 31;
  if (row >= n) return;
  const int id = ids[row];
  const bool ok = id >= 0 && id < vocab;
  if (!ok && lane == 0) set_device_error(err, DEVERR_INDEX);
  const int nv = d / V;
  for (int c = lane; c < nv; c += 32) {
    uint4 u = ok ? *reinterpret_cast<const uint4*>(table + (int64_t)id * d + c * V)
                 : make_uint4(0, 0, 0, 0);
    *reinterpret_cast<uint4*>(out + row * d + c * V) = u;
  }
}

// ---------------------------------------------------------------- gather + norm
// Norm parameters (g1, b1, g2, b2; biases absent for RMSNorm, second pair
// absent without out2) staged once per block in shared memory, so that the
// per-row loop reads them without waiting behind its own global stores.
template <typename T>
__device__ __forceinline__ void stage_norm_params(const T* g1, const T* b1, const T* g2, const T* b2,
                                                  int d, T* sp) {
  constexpr int V = Elem<T>::kVec;
  const int nv = d / V;
  const T* src[4] = {g1, b1, g2, b2};
  for (int k = 0; k < 4; ++k) {
    if (!src[k]) continue;
    for (int i = threadIdx.x; i < nv; i += blockDim.x)
      reinterpret_cast<uint4*>(sp + k * d)[i] = reinterpret_cast<const uint4*>(src[k])[i];
  }
  __syncthreads();
}

// o1 = norm(xr; g1, b1), o2 = norm(xr; g2, b2) for R rows at once (their
// loads overlap), by one warp; row r is skipped when xr[r] is null. NCH: the
// 16-byte vectors per lane a row needs, ceil(d / (32 V)), fixed at compile
// time so that no dead chunk is issued. sp holds the staged parameters
// ([4][d]: g1, b1, g2, b2). LayerNorm: (x - mean) / sqrt(var + eps) * g + b
// (biased variance, two-pass over the register-resident row); RMSNorm:
// x / sqrt(mean(x^2) + eps) * g.
template <typename T, bool RMS, int NCH, int R>
__device__ __forceinline__ void norm_rows(const T* const (&xr)[R], int d, const T* sp, float eps,
                                          T* const (&o1)[R], T* const (&o2)[R], int lane) {
  constexpr int V = Elem<T>::kVec;
  const int nv = d / V;
  float v[R][NCH][V];
  float s[R], mean[R], rstd[R];
#pragma unroll
  for (int r = 0; r < R; ++r) {
    s[r] = 0.f;
    if (!xr[r]) continue;
#pragma unroll
    for (int c = 0; c < NCH; ++c) {
      const int ci = c * 32 + lane;
      if (ci < nv) load_vec(xr[r] + ci * V, v[r][c]);
    }
  }
#pragma unroll
  for (int r = 0; r < R; ++r) {
#pragma unroll
    for (int c = 0; c < NCH; ++c) {
      const int ci = c * 32 + lane;
      if (xr[r] && ci < nv) {
#pragma unroll
        for (int j = 0; j < V; ++j) s[r] += RMS ? v[r][c][j] * v[r][c][j] : v[r][c][j];
      }
    }
  }
#pragma unroll
  for (int r = 0; r < R; ++r) {
    if (RMS) {
      mean[r] = 0.f;
      rstd[r] = 1.f / sqrtf(warp_sum(s[r]) / d + eps);
    } else {
      mean[r] = warp_sum(s[r]) / d;
    }
  }
  if (!RMS) {
#pragma unroll
    for (int r = 0; r < R; ++r) {
      float q = 0.f;
#pragma unroll
      for (int c = 0; c < NCH; ++c) {
        const int ci = c * 32 + lane;
        if (xr[r] && ci < nv) {
#pragma unroll
          for (int j = 0; j < V; ++j) {
            const float t = v[r][c][j] - mean[r];
            q += t * t;
          }
        }
      }
      rstd[r] = 1.f / sqrtf(warp_sum(q) / d + eps);
    }
  }
#pragma unroll
  for (int c = 0; c < NCH; ++c) {
    const int ci = c * 32 + lane;
    if (ci < nv) {
      float g[V], bb[V], o[V];
      load_vec(sp + ci * V, g);
      if (!RMS) load_vec(sp + d + ci * V, bb);
#pragma unroll
      for (int r = 0; r < R; ++r) {
        if (!xr[r]) continue;
#pragma unroll
        for (int j = 0; j < V; ++j)
          o[j] = (v[r][c][j] - mean[r]) * rstd[r] * g[j] + (RMS ? 0.f : bb[j]);
        store_vec(o1[r] + ci * V, o);
      }
      if (o2[0]) {
        load_vec(sp + 2 * d + ci * V, g);
        if (!RMS) load_vec(sp + 3 * d + ci * V, bb);
#pragma unroll
        for (int r = 0; r < R; ++r) {
          if (!xr[r]) continue;
#pragma unroll
          for (int j = 0; j < V; ++j)
            o[j] = (v[r][c][j] - mean[r]) * rstd[r] * g[j] + (RMS ? 0.f : bb[j]);
          store_vec(o2[r] + ci * V, o);
        }
      }
    }
  }
}

// Rows per step of one warp: two while a row needs at most 8 vectors per lane.
template <int NCH>
constexpr int rows_per_step() { return NCH <= 8 ? 2 : 1; }

// Rows [lo, hi) of the block's share, warp w taking w, w + nw, ... in steps
// of R rows; src(i) / dst(i) give the source row and the output row.
template <typename T, bool RMS, int NCH, typename Src, typename Dst>
__device__ __forceinline__ void norm_share(int64_t lo, int64_t hi, const T* x, int d, const T* sp,
                                           float eps, T* out1, T* out2, Src src, Dst dst) {
  constexpr int R = rows_per_step<NCH>();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  for (int64_t i = lo + warp; i < hi; i += (int64_t)R * nw) {
    const T* xr[R];
    T* o1[R];
    T* o2[R];
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const int64_t ii = i + (int64_t)r * nw;
      const bool ok = ii < hi;
      const int64_t m = ok ? dst(ii) : 0;
      xr[r] = ok ? x + src(ii) * d : nullptr;
      o1[r] = out1 + m * d;
      o2[r] = out2 ? out2 + m * d : nullptr;
    }
    norm_rows<T, RMS, NCH, R>(xr, d, sp, eps, o1, o2, lane);
  }
}

// ---------------------------------------------------------------- few rows
// Gather + norm of a few rows (a decode step's one row per sequence): four
// warps per block, one row per warp, the row in registers; the parameters
// are staged before waiting for the previous kernel (they do not depend on it).
constexpr int kFewRowWarps = 4;
constexpr int64_t kFewRowsMax = 512;   // larger counts stream through gather_norm_tma_kernel

template <typename T, bool RMS, int NCH>
__global__ void __launch_bounds__(32 * kFewRowWarps)
    norm_few_rows_kernel(const T* x, const int32_t* rows, int64_t M, int d, const T* g1, const T* b1,
                         const T* g2, const T* b2, float eps, T* out1, T* out2) {
  pdl_trigger();
  extern __shared__ __align__(16) uint8_t smem_few[];
  T* sp = reinterpret_cast<T*>(smem_few);
  stage_norm_params(g1, RMS ? nullptr : b1, out2 ? g2 : nullptr, (RMS || !out2) ? nullptr : b2, d, sp);
  pdl_wait();
  const int64_t lo = (int64_t)blockIdx.x * kFewRowWarps;
  const int64_t hi = lo + kFewRowWarps < M ? lo + kFewRowWarps : M;
  norm_share<T, RMS, NCH>(
      lo, hi, x, d, sp, eps, out1, out2, [&](int64_t i) { return rows ? (int64_t)rows[i] : i; },
      [&](int64_t i) { return i; });
}

// A decode step's first pass: the norm(s) of the B new rows (one per
// sequence) as above, and each row's keep decision at this layer (lane 0 of
// its warp): kept iff its router score is above the layer's threshold (a tie
// loses, NaN never wins); rows[b] = b if kept, else -1 (the residual scatter
// skips it); pos[b] = the current position from the cache header. A cache
// not filled by a prefill of this shape, or a position past its rotary
// table, raises DEVERR_INDEX and the position is clamped into range.
template <typename T, bool RMS, int NCH>
__global__ void __launch_bounds__(32 * kFewRowWarps)
    decide_norm_kernel(const T* x, int B, int d, const T* g1, const T* b1, const T* g2, const T* b2, float eps,
                       T* out1, T* out2, const float* scores, const float* thr, const int32_t* hdr, int C_max,
                       int32_t* rows, int32_t* pos, int32_t* kept_out, int* err) {
  pdl_trigger();
  extern __shared__ __align__(16) uint8_t smem_dn[];
  T* sp = reinterpret_cast<T*>(smem_dn);
  stage_norm_params(g1, RMS ? nullptr : b1, out2 ? g2 : nullptr, (RMS || !out2) ? nullptr : b2, d, sp);
  pdl_wait();
  const int64_t lo = (int64_t)blockIdx.x * kFewRowWarps;
  const int64_t hi = lo + kFewRowWarps < B ? lo + kFewRowWarps : B;
  const int b = (int)lo + (int)(threadIdx.x >> 5);
  if (b < hi && (threadIdx.x & 31) == 0) {
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
  norm_share<T, RMS, NCH>(lo, hi, x, d, sp, eps, out1, out2, [](int64_t i) { return i; },
                          [](int64_t i) { return i; });
}

// ---------------------------------------------------------------- TMA-staged gather + norm
// For large row counts (HBM bound): one warp streams whole source rows into a
// shared-memory ring with one bulk copy each (cp.async.bulk, completion on the
// slot's mbarrier), eight warps normalise them from shared memory, one warp
// per row, and release the slot. Many rows are in flight per SM with few
// registers, and each 16-byte global store of a warp covers 512 contiguous
// bytes of an output row.
constexpr int kRowWarps = 8;                       // consumer warps
constexpr int kRowThreads = 32 * (kRowWarps + 1);  // + the producer warp
constexpr int kRowSlots = 16;                      // ring slots (two rows per consumer warp)
static_assert(kRowSlots % kRowWarps == 0, "a slot is always consumed by the same warp");
constexpr int kMaxRowBytes = 8192;   // d <= 4096 (bf16) or 2048 (fp32)

// A 16-byte vector as V / 2 pairs of floats, and back (round to nearest even).
__device__ __forceinline__ void unpack_pairs(const uint4& u, float2* p, bf16) {
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) p[i] = make_float2(__uint_as_float(w[i] << 16), __uint_as_float(w[i] & 0xffff0000u));
}
__device__ __forceinline__ void unpack_pairs(const uint4& u, float2* p, float) {
  p[0] = make_float2(__uint_as_float(u.x), __uint_as_float(u.y));
  p[1] = make_float2(__uint_as_float(u.z), __uint_as_float(u.w));
}
__device__ __forceinline__ uint4 pack_pairs(const float2* p, bf16) {
  return make_uint4(pack_bf16x2(p[0].x, p[0].y), pack_bf16x2(p[1].x, p[1].y), pack_bf16x2(p[2].x, p[2].y),
                    pack_bf16x2(p[3].x, p[3].y));
}
__device__ __forceinline__ uint4 pack_pairs(const float2* p, float) {
  return make_uint4(__float_as_uint(p[0].x), __float_as_uint(p[0].y), __float_as_uint(p[1].x),
                    __float_as_uint(p[1].y));
}

// out1[m] = norm(x[row(m)]; g1, b1), out2[m] = norm(x[row(m)]; g2, b2) for the
// block's contiguous share of m. Shared memory: the staged parameters
// ([4][d]), then the ring (kRowSlots rows of d), then 2 kRowSlots mbarriers.
// NCH: the 16-byte vectors of a row per lane, ceil(d / (32 V)) rounded up to
// a compiled bucket: a consumer warp holds its row in registers (one shared-
// memory read of the slot) and works on pairs of floats.
template <typename T, bool RMS, int NCH>
__global__ void __launch_bounds__(kRowThreads)
    gather_norm_tma_kernel(const T* x, const int32_t* rows, int64_t M, int d, const T* g1,
                           const T* b1, const T* g2, const T* b2, float eps, T* out1, T* out2,
                           int* err, unsigned long long timeout_ns) {
  pdl_trigger();
  extern __shared__ __align__(16) uint8_t smem_rows[];
  constexpr int V = Elem<T>::kVec;
  const uint32_t row_bytes = (uint32_t)d * sizeof(T);
  T* sp = reinterpret_cast<T*>(smem_rows);
  uint8_t* ring = smem_rows + 4 * (size_t)row_bytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(ring + (size_t)kRowSlots * row_bytes);
  const uint32_t full0 = smem_u32(bars), empty0 = full0 + 8 * kRowSlots;
  __shared__ int abort_flag;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kRowSlots; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    abort_flag = 0;
    fence_barrier_init();
  }
  stage_norm_params(g1, RMS ? nullptr : b1, out2 ? g2 : nullptr, (RMS || !out2) ? nullptr : b2, d,
                    sp);   // weights: independent of the previous kernel (also syncs the block)
  pdl_wait();
  const int64_t lo = (int64_t)blockIdx.x * M / gridDim.x, hi = (int64_t)(blockIdx.x + 1) * M / gridDim.x;
  const int64_t n = hi - lo;
  volatile int* abort_v = &abort_flag;

  if (warp == kRowWarps) {
    // ------------------------------------------------------------ producer
    // The warp reads the source row indices 32 at a time; lane 0 issues the copies.
    int64_t issued = 0;
    bool ok = true;
    for (int64_t j0 = 0; j0 < n && ok; j0 += 32) {
      int64_t src_l = 0;
      if (j0 + lane < n) src_l = rows ? (int64_t)rows[lo + j0 + lane] : lo + j0 + lane;
      const int cnt = (int)(n - j0 < 32 ? n - j0 : 32);
      for (int k = 0; k < cnt; ++k) {
        const int64_t src = __shfl_sync(0xffffffffu, src_l, k);
        const int64_t j = j0 + k;
        const int s = (int)(j % kRowSlots);
        const uint32_t round = (uint32_t)(j / kRowSlots);
        int w = 1;
        if (lane == 0) {
          if (round > 0)
            w = mbar_wait_bounded(empty0 + 8 * s, (round - 1) & 1, abort_v, err, timeout_ns);
          if (w) {
            mbar_arrive_expect_tx(full0 + 8 * s, row_bytes);
            bulk_load(smem_u32(ring + (size_t)s * row_bytes), x + src * d, row_bytes, full0 + 8 * s);
          }
        }
        if (!__shfl_sync(0xffffffffu, w, 0)) {
          ok = false;
          break;
        }
        ++issued;
      }
    }
    // every copy issued has landed before the block may exit
    if (lane == 0)
      for (int s = 0; s < kRowSlots && s < issued; ++s) {
        const int64_t last = s + ((issued - 1 - s) / kRowSlots) * kRowSlots;
        mbar_wait_drain(full0 + 8 * s, (uint32_t)((last / kRowSlots) & 1), timeout_ns);
      }
  } else {
    // ------------------------------------------------------------ consumers
    constexpr int P = V / 2;                    // float pairs per vector
    const int nv = d / V;
    const float inv_d = 1.f / (float)d;
    for (int64_t j = warp; j < n; j += kRowWarps) {
      const int s = (int)(j % kRowSlots);
      int ok = 0;
      if (lane == 0)
        ok = mbar_wait_bounded(full0 + 8 * s, (uint32_t)((j / kRowSlots) & 1), abort_v, err, timeout_ns);
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) break;
      const uint4* xr = reinterpret_cast<const uint4*>(ring + (size_t)s * row_bytes);
      uint4 raw[NCH];
#pragma unroll
      for (int c = 0; c < NCH; ++c)
        if (c * 32 + lane < nv) raw[c] = xr[c * 32 + lane];
      // statistics over pairs (two partial sums), then over the warp
      float2 acc = make_float2(0.f, 0.f);
#pragma unroll
      for (int c = 0; c < NCH; ++c) {
        if (c * 32 + lane < nv) {
          float2 f[P];
          unpack_pairs(raw[c], f, T());
#pragma unroll
          for (int k = 0; k < P; ++k) acc = RMS ? __ffma2_rn(f[k], f[k], acc) : __fadd2_rn(acc, f[k]);
        }
      }
      // every value of the slot has been used: it may be refilled
      __syncwarp();
      if (lane == 0) mbar_arrive(empty0 + 8 * s);
      float mean = 0.f, rstd;
      if (RMS) {
        rstd = 1.f / sqrtf(warp_sum(acc.x + acc.y) * inv_d + eps);
      } else {
        mean = warp_sum(acc.x + acc.y) * inv_d;
        const float2 negm = make_float2(-mean, -mean);
        float2 q = make_float2(0.f, 0.f);
#pragma unroll
        for (int c = 0; c < NCH; ++c) {
          if (c * 32 + lane < nv) {
            float2 f[P];
            unpack_pairs(raw[c], f, T());
#pragma unroll
            for (int k = 0; k < P; ++k) {
              const float2 t = __fadd2_rn(f[k], negm);
              q = __ffma2_rn(t, t, q);
            }
          }
        }
        rstd = 1.f / sqrtf(warp_sum(q.x + q.y) * inv_d + eps);
      }
      const float2 negm = make_float2(-mean, -mean), rs = make_float2(rstd, rstd);
      const int64_t m = lo + j;
#pragma unroll
      for (int c = 0; c < NCH; ++c) {
        const int ci = c * 32 + lane;
        if (ci < nv) {
          float2 f[P], g[P], bb[P], o[P];
          unpack_pairs(raw[c], f, T());
#pragma unroll
          for (int k = 0; k < P; ++k) f[k] = __fmul2_rn(RMS ? f[k] : __fadd2_rn(f[k], negm), rs);
          unpack_pairs(reinterpret_cast<const uint4*>(sp)[ci], g, T());
          if (!RMS) unpack_pairs(reinterpret_cast<const uint4*>(sp + d)[ci], bb, T());
#pragma unroll
          for (int k = 0; k < P; ++k) o[k] = RMS ? __fmul2_rn(f[k], g[k]) : __ffma2_rn(f[k], g[k], bb[k]);
          reinterpret_cast<uint4*>(out1 + m * d)[ci] = pack_pairs(o, T());
          if (out2) {
            unpack_pairs(reinterpret_cast<const uint4*>(sp + 2 * d)[ci], g, T());
            if (!RMS) unpack_pairs(reinterpret_cast<const uint4*>(sp + 3 * d)[ci], bb, T());
#pragma unroll
            for (int k = 0; k < P; ++k) o[k] = RMS ? __fmul2_rn(f[k], g[k]) : __ffma2_rn(f[k], g[k], bb[k]);
            reinterpret_cast<uint4*>(out2 + m * d)[ci] = pack_pairs(o, T());
          }
        }
      }
    }
  }
}

// ---------------------------------------------------------------- rotary embedding
// tab[p * half + i] = (cos, sin) of the angle p * inv[i], inv[i] =
// theta^(-2i / rotary_dim) given in fp64 by the host. The angle is formed and
// reduced to [-pi, pi] in fp64, then evaluated in fp32 (error ~1e-7).
struct InvFreq {
  double v[64];
};
__global__ void rope_table_kernel(float2* tab, int T, int half, InvFreq inv) {
  pdl_trigger();
  pdl_wait();
  const int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (k >= (int64_t)T * half) return;
  const int p = (int)(k / half), i = (int)(k % half);
  double a = (double)p * inv.v[i];
  a -= rint(a * 0.15915494309189535) * 6.283185307179586;
  float s, c;
  sincosf((float)a, &s, &c);
  tab[k] = make_float2(c, s);
}

// Rotates, in place, the first rotary_dim features of every query and key
// head of row m at position pos[m] (or m % T when pos is null): feature i pairs
// with i + rotary_dim/2.
template <typename T>
__global__ void rope_apply_kernel(T* qkv, int64_t M, int64_t ld, int heads, int head_dim,
                                  int half, const int32_t* pos, int seq_len, const float2* tab) {
  pdl_trigger();
  pdl_wait();
  const int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t per_row = (int64_t)heads * half;
  if (k >= M * per_row) return;
  const int64_t m = k / per_row;
  const int r = (int)(k % per_row);
  const int h = r / half, i = r % half;
  const int p = pos ? pos[m] : (int)(m % seq_len);
  const float2 cs = tab[(int64_t)p * half + i];
  T* base = qkv + m * ld + (int64_t)h * head_dim;
  const float a = Elem<T>::to_f(base[i]);
  const float b = Elem<T>::to_f(base[i + half]);
  base[i] = Elem<T>::from_f(a * cs.x - b * cs.y);
  base[i + half] = Elem<T>::from_f(b * cs.x + a * cs.y);
}

// ---------------------------------------------------------------- fp32 router (Sec. 3.4)
// One warp per token: score = sum_j w2[j] * silu(w1[j] . x + b1[j]) + b2.
__global__ void router_f32_kernel(const float* x, int64_t n, int d, int h, const float* w1,
                                  const float* b1, const float* w2, const float* b2,
                                  float* scores) {
  pdl_trigger();
  pdl_wait();
  const int64_t row = (int64_t)blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
  const int lane = threadIdx.x & 31;
  if (row >= n) return;
  const float* xr = x + row * d;
  float s = 0.f;
  for (int j = 0; j < h; ++j) {
    const float* wr = w1 + (int64_t)j * d;
    float dot = 0.f;
    for (int c = lane * 4; c < d; c += 128) {
      const float4 a = *reinterpret_cast<const float4*>(xr + c);
      const float4 b = *reinterpret_cast<const float4*>(wr + c);
      dot = fmaf(a.x, b.x, fmaf(a.y, b.y, fmaf(a.z, b.z, fmaf(a.w, b.w, dot))));
    }
    const float u = warp_sum(dot) + b1[j];
    s += w2[j] * (u / (1.f + expf(-u)));
  }
  if (lane == 0) scores[row] = s + b2[0];
}

// ---------------------------------------------------------------- Top-K (Sec. 3.4)
// (radix select and emission: topk.cuh)
constexpr int kTopkThreads = 1024;

// One block per sequence: idx[b][i] = i-th kept position (ascending), rows[b][i] = b T + position.
__global__ void __launch_bounds__(kTopkThreads) topk_kernel(const float* scores, int T, int K,
                                                            int32_t* idx, int32_t* rows) {
  pdl_trigger();
  pdl_wait();
  extern __shared__ uint32_t keys[];
  __shared__ TopkShared sh;
  const int b = blockIdx.x;
  const float* sc = scores + (int64_t)b * T;
  for (int t = threadIdx.x; t < T; t += kTopkThreads) keys[t] = score_key(sc[t]);
  uint32_t kth;
  int need_eq;
  const auto sync = [] { __syncthreads(); };
  radix_select<kTopkThreads>(keys, T, K, sh, kth, need_eq, (int)threadIdx.x, sync);
  emit_kept<kTopkThreads>(keys, T, kth, need_eq, sh, (int)threadIdx.x, sync, [&](int i, int t) {
    idx[(int64_t)b * K + i] = t;
    if (rows) rows[(int64_t)b * K + i] = b * T + t;
  });
}

constexpr int kSelThreads = 256;

// Top-K of sequence b fused with the gather and norm of its kept rows: every
// block of the sequence selects the same kept set (deterministic) into shared
// memory, then normalises its share [g K / G, (g+1) K / G) of the packed rows
// (one warp per row) and writes that share of idx / rows.
template <typename T, bool RMS, int NCH>
__global__ void __launch_bounds__(kSelThreads)
    select_gather_norm_kernel(const float* scores, int Tlen, int K, const T* x, int d, const T* g1,
                              const T* b1, const T* g2, const T* b2, float eps, T* out1, T* out2,
                              int32_t* idx, int32_t* rows) {
  pdl_trigger();
  extern __shared__ __align__(16) uint32_t smem_sel[];
  T* sp = reinterpret_cast<T*>(smem_sel);                               // [4][d] norm parameters
  uint32_t* keys = smem_sel + (4 * d * sizeof(T)) / 4;                  // [Tlen]
  int32_t* kept = reinterpret_cast<int32_t*>(keys + Tlen);              // [K]
  __shared__ TopkShared sh;
  stage_norm_params(g1, RMS ? nullptr : b1, out2 ? g2 : nullptr, (RMS || !out2) ? nullptr : b2, d,
                    sp);   // weights: independent of the previous kernel
  pdl_wait();
  const int b = blockIdx.y, g = blockIdx.x, G = gridDim.x;
  const float* sc = scores + (int64_t)b * Tlen;
  for (int t = threadIdx.x; t < Tlen; t += kSelThreads) keys[t] = score_key(sc[t]);
  uint32_t kth;
  int need_eq;
  const auto sync = [] { __syncthreads(); };
  radix_select<kSelThreads>(keys, Tlen, K, sh, kth, need_eq, (int)threadIdx.x, sync);
  emit_kept<kSelThreads>(keys, Tlen, kth, need_eq, sh, (int)threadIdx.x, sync,
                         [&](int i, int t) { kept[i] = t; });
  __syncthreads();
  const int lo = (int)((int64_t)g * K / G), hi = (int)((int64_t)(g + 1) * K / G);
  for (int i = lo + (int)threadIdx.x; i < hi; i += kSelThreads) {
    idx[(int64_t)b * K + i] = kept[i];
    rows[(int64_t)b * K + i] = b * Tlen + kept[i];
  }
  norm_share<T, RMS, NCH>(
      lo, hi, x, d, sp, eps, out1, out2, [&](int64_t i) { return (int64_t)b * Tlen + kept[i]; },
      [&](int64_t i) { return (int64_t)b * K + i; });
}

// ---------------------------------------------------------------- Eq. 4 statistics
constexpr int kStatThreads = 256;

// One warp per row: fp32 sums a.b, |a|^2, |b|^2; per block fixed-order fp64
// sums of either the row cosines (TOKEN) or the three sums (FLAT).
template <typename T>
__global__ void __launch_bounds__(kStatThreads) cos_rows_kernel(const T* a, const T* b,
                                                                int64_t n_rows, int d, int mode,
                                                                double* partials) {
  pdl_trigger();
  pdl_wait();
  constexpr int V = Elem<T>::kVec;
  __shared__ double red[kStatThreads / 32][3];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int64_t nwarps = (int64_t)gridDim.x * (kStatThreads / 32);
  double acc0 = 0, acc1 = 0, acc2 = 0;
  for (int64_t r = (int64_t)blockIdx.x * (kStatThreads / 32) + w; r < n_rows; r += nwarps) {
    float dot = 0.f, na = 0.f, nb = 0.f;
    for (int c = lane * V; c < d; c += 32 * V) {
      float fa[V], fb[V];
      load_vec(a + r * d + c, fa);
      load_vec(b + r * d + c, fb);
#pragma unroll
      for (int j = 0; j < V; ++j) {
        dot = fmaf(fa[j], fb[j], dot);
        na = fmaf(fa[j], fa[j], na);
        nb = fmaf(fb[j], fb[j], nb);
      }
    }
    dot = warp_sum(dot);
    na = warp_sum(na);
    nb = warp_sum(nb);
    if (mode == 0) {
      const double den = fmax(sqrt((double)na), 1e-8) * fmax(sqrt((double)nb), 1e-8);
      acc0 += (double)dot / den;
    } else {
      acc0 += dot; acc1 += na; acc2 += nb;
    }
  }
  if (lane == 0) { red[w][0] = acc0; red[w][1] = acc1; red[w][2] = acc2; }
  __syncthreads();
  if (threadIdx.x < 3) {
    double s = 0;
    for (int i = 0; i < kStatThreads / 32; ++i) s += red[i][threadIdx.x];
    partials[(int64_t)blockIdx.x * 3 + threadIdx.x] = s;
  }
}

// Eq. 4 from per-chunk partials {a.b, |a|^2, |b|^2} ([n_rows][nch] float4,
// written by a projection epilogue): one warp per row sums its chunks (fp32,
// fixed lane order), then the same per-block fixed-order fp64 sums as
// cos_rows_kernel.
__global__ void __launch_bounds__(kStatThreads) cos_chunks_kernel(const float4* parts, int64_t n_rows,
                                                                  int nch, int mode, double* partials) {
  pdl_trigger();
  pdl_wait();
  __shared__ double red[kStatThreads / 32][3];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int64_t nwarps = (int64_t)gridDim.x * (kStatThreads / 32);
  double acc0 = 0, acc1 = 0, acc2 = 0;
  for (int64_t r = (int64_t)blockIdx.x * (kStatThreads / 32) + w; r < n_rows; r += nwarps) {
    float dot = 0.f, na = 0.f, nb = 0.f;
    for (int c = lane; c < nch; c += 32) {
      const float4 f = parts[r * nch + c];
      dot += f.x;
      na += f.y;
      nb += f.z;
    }
    dot = warp_sum(dot);
    na = warp_sum(na);
    nb = warp_sum(nb);
    if (mode == 0) {
      const double den = fmax(sqrt((double)na), 1e-8) * fmax(sqrt((double)nb), 1e-8);
      acc0 += (double)dot / den;
    } else {
      acc0 += dot; acc1 += na; acc2 += nb;
    }
  }
  if (lane == 0) { red[w][0] = acc0; red[w][1] = acc1; red[w][2] = acc2; }
  __syncthreads();
  if (threadIdx.x < 3) {
    double s = 0;
    for (int i = 0; i < kStatThreads / 32; ++i) s += red[i][threadIdx.x];
    partials[(int64_t)blockIdx.x * 3 + threadIdx.x] = s;
  }
}

// Fixed-order sum of the per-block partials, added to acc.
__global__ void cos_finish_kernel(const double* partials, int nblocks, int64_t n_rows, int mode,
                                  double* acc) {
  pdl_trigger();
  pdl_wait();
  __shared__ double red[3][256];
  double s[3] = {0, 0, 0};
  for (int i = threadIdx.x; i < nblocks; i += 256)
    for (int j = 0; j < 3; ++j) s[j] += partials[(int64_t)i * 3 + j];
  for (int j = 0; j < 3; ++j) red[j][threadIdx.x] = s[j];
  __syncthreads();
  for (int o = 128; o > 0; o >>= 1) {
    if (threadIdx.x < o)
      for (int j = 0; j < 3; ++j) red[j][threadIdx.x] += red[j][threadIdx.x + o];
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    if (mode == 0) {
      acc[0] += red[0][0];
      acc[1] += (double)n_rows;
    } else {
      acc[0] += red[0][0]; acc[1] += red[1][0]; acc[2] += red[2][0];
    }
  }
}

// Fixed scratch of the workspace-free statistics entry point: one slot of
// three doubles per reduction block. The block count never exceeds
// kStatMaxBlocks (see stats_partials_count), so 48 KiB always suffice.
constexpr int kStatMaxBlocks = 2048;
static __device__ __align__(256) double g_stats_scratch[kStatMaxBlocks * 3];

// idx[b * K + j] = j: the kept positions of a dense layer.
__global__ void iota_kernel(int32_t* idx, int64_t n, int K) {
  pdl_trigger();
  pdl_wait();
  const int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (k < n) idx[k] = (int32_t)(k % K);
}

// ---------------------------------------------------------------- bounded-wait self-test
__global__ void bounded_wait_selftest_kernel(int* err, unsigned long long timeout_ns) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(smem_u32(&bar), 1);
    abort_flag = 0;
    fence_barrier_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    // Nothing ever arrives: the wait must give up and flag the error word.
    mbar_wait_bounded(smem_u32(&bar), 0, &abort_flag, err, timeout_ns);
  }
  __syncthreads();
}

}  // namespace

// ---------------------------------------------------------------- launchers
static unsigned blocks_for(int64_t rows, int rows_per_block) {
  return (unsigned)((rows + rows_per_block - 1) / rows_per_block);
}

cudaError_t embed(int dtype, const int32_t* ids, int64_t n, const void* table, int vocab, int d,
                  void* out, const Dev& dev) {
  if (n <= 0) return cudaSuccess;
  if (dtype == kBF16)
    return launch_pdl(embed_kernel<bf16>, dim3(blocks_for(n, 8)), dim3(256), 0, dev.stream, ids, n,
                      static_cast<const bf16*>(table), vocab, d, static_cast<bf16*>(out), dev.err);
  return launch_pdl(embed_kernel<float>, dim3(blocks_for(n, 8)), dim3(256), 0, dev.stream, ids, n,
                    static_cast<const float*>(table), vocab, d, static_cast<float*>(out), dev.err);
}

// Chunk-count bucket (vectors per lane) of a row of d elements.
template <typename T>
int nch_bucket(int d) {
  const int n = (d / Elem<T>::kVec + 31) / 32;
  if (n <= 2) return 2;
  if (n <= 4) return n;
  if (n <= 6) return 6;
  if (n <= 8) return 8;
  if (n <= 12) return 12;
  if (n <= 14) return 14;
  return 16;
}

// Calls f(std::integral_constant<int, NCH>) for the bucket of d.
template <typename T, typename F>
cudaError_t with_nch(int d, F f) {
  switch (nch_bucket<T>(d)) {
    case 2: return f(std::integral_constant<int, 2>());
    case 3: return f(std::integral_constant<int, 3>());
    case 4: return f(std::integral_constant<int, 4>());
    case 6: return f(std::integral_constant<int, 6>());
    case 8: return f(std::integral_constant<int, 8>());
    case 12: return f(std::integral_constant<int, 12>());
    case 14: return f(std::integral_constant<int, 14>());
    default: return f(std::integral_constant<int, 16>());
  }
}

template <typename T, bool RMS, int NCH>
cudaError_t gather_norm_launch(const void* x, const int32_t* rows, int64_t M, int d, const void* g1,
                               const void* b1, const void* g2, const void* b2, float eps, void* out1,
                               void* out2, const Dev& dev) {
  const size_t row_bytes = (size_t)d * sizeof(T);
  const size_t smem = 4 * row_bytes + kRowSlots * row_bytes + 2 * kRowSlots * 8;
  static int attr_done[64] = {0};
  int device = 0;
  cudaGetDevice(&device);
  if (device < 64 && !attr_done[device]) {
    cudaError_t e = cudaFuncSetAttribute(gather_norm_tma_kernel<T, RMS, NCH>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (4 + kRowSlots) * kMaxRowBytes + 2 * kRowSlots * 8);
    if (e != cudaSuccess) return e;
    attr_done[device] = 1;
  }
  // one wave: as many blocks per SM as fit (at most two), at least one row
  // per consumer warp
  const int64_t fit = std::max<int64_t>(1, std::min<int64_t>(2, 232448 / (int64_t)(smem + 1024)));
  const int64_t grid = std::max<int64_t>(1, std::min<int64_t>((M + kRowWarps - 1) / kRowWarps,
                                                             fit * dev.num_sms));
  return launch_pdl(gather_norm_tma_kernel<T, RMS, NCH>, dim3((unsigned)grid), dim3(kRowThreads), smem,
                    dev.stream, static_cast<const T*>(x), rows, M, d, static_cast<const T*>(g1),
                    static_cast<const T*>(b1), static_cast<const T*>(g2),
                    static_cast<const T*>(b2), eps, static_cast<T*>(out1), static_cast<T*>(out2),
                    dev.err, kWaitTimeoutNs);
}

template <typename T, bool RMS>
cudaError_t gather_norm_t(const void* x, const int32_t* rows, int64_t M, int d, const void* g1,
                          const void* b1, const void* g2, const void* b2, float eps, void* out1,
                          void* out2, const Dev& dev) {
  return with_nch<T>(d, [&](auto nch) {
    constexpr int NCH = decltype(nch)::value;
    if (M <= kFewRowsMax)
      return launch_pdl(norm_few_rows_kernel<T, RMS, NCH>, dim3((unsigned)((M + kFewRowWarps - 1) / kFewRowWarps)),
                        dim3(32 * kFewRowWarps), 4 * (size_t)d * sizeof(T), dev.stream, static_cast<const T*>(x), rows,
                        M, d, static_cast<const T*>(g1), static_cast<const T*>(b1), static_cast<const T*>(g2),
                        static_cast<const T*>(b2), eps, static_cast<T*>(out1), static_cast<T*>(out2));
    return gather_norm_launch<T, RMS, NCH>(x, rows, M, d, g1, b1, g2, b2, eps, out1, out2, dev);
  });
}

template <typename T, bool RMS>
cudaError_t decide_norm_t(const void* x, int B, int d, const void* g1, const void* b1, const void* g2,
                          const void* b2, float eps, void* out1, void* out2, const float* scores, const float* thr,
                          const int32_t* hdr, int C_max, int32_t* rows, int32_t* pos, int32_t* kept_out,
                          const Dev& dev) {
  return with_nch<T>(d, [&](auto nch) {
    return launch_pdl(decide_norm_kernel<T, RMS, decltype(nch)::value>,
                      dim3((unsigned)((B + kFewRowWarps - 1) / kFewRowWarps)), dim3(32 * kFewRowWarps),
                      4 * (size_t)d * sizeof(T), dev.stream, static_cast<const T*>(x), B, d,
                      static_cast<const T*>(g1), static_cast<const T*>(b1), static_cast<const T*>(g2),
                      static_cast<const T*>(b2), eps, static_cast<T*>(out1), static_cast<T*>(out2), scores, thr,
                      hdr, C_max, rows, pos, kept_out, dev.err);
  });
}

cudaError_t decide_norm(int dtype, const void* x, int B, int d, bool is_rms, const void* g1, const void* b1,
                        const void* g2, const void* b2, float eps, void* out1, void* out2, const float* scores,
                        const float* thr, const int32_t* hdr, int C_max, int32_t* rows, int32_t* pos,
                        int32_t* kept_out, const Dev& dev) {
  if (B <= 0) return cudaSuccess;
  if (dtype == kBF16)
    return is_rms ? decide_norm_t<bf16, true>(x, B, d, g1, b1, g2, b2, eps, out1, out2, scores, thr, hdr, C_max,
                                               rows, pos, kept_out, dev)
                  : decide_norm_t<bf16, false>(x, B, d, g1, b1, g2, b2, eps, out1, out2, scores, thr, hdr, C_max,
                                                rows, pos, kept_out, dev);
  return is_rms ? decide_norm_t<float, true>(x, B, d, g1, b1, g2, b2, eps, out1, out2, scores, thr, hdr, C_max,
                                              rows, pos, kept_out, dev)
                : decide_norm_t<float, false>(x, B, d, g1, b1, g2, b2, eps, out1, out2, scores, thr, hdr, C_max,
                                               rows, pos, kept_out, dev);
}

cudaError_t gather_norm(int dtype, const void* x, const int32_t* rows, int64_t M, int d,
                        bool is_rms, const void* g1, const void* b1, const void* g2,
                        const void* b2, float eps, void* out1, void* out2, const Dev& dev) {
  if (M <= 0) return cudaSuccess;
  if (dtype == kBF16)
    return is_rms ? gather_norm_t<bf16, true>(x, rows, M, d, g1, b1, g2, b2, eps, out1, out2, dev)
                  : gather_norm_t<bf16, false>(x, rows, M, d, g1, b1, g2, b2, eps, out1, out2, dev);
  return is_rms ? gather_norm_t<float, true>(x, rows, M, d, g1, b1, g2, b2, eps, out1, out2, dev)
                : gather_norm_t<float, false>(x, rows, M, d, g1, b1, g2, b2, eps, out1, out2, dev);
}

cudaError_t rope_table(float2* tab, int T, int rotary_dim, float theta, const Dev& dev) {
  const int half = rotary_dim / 2;
  const int64_t n = (int64_t)T * half;
  if (n <= 0) return cudaSuccess;
  if (half > 64) return cudaErrorInvalidValue;
  InvFreq inv;
  for (int i = 0; i < 64; ++i) inv.v[i] = i < half ? pow((double)theta, -2.0 * i / rotary_dim) : 0.0;
  return launch_pdl(rope_table_kernel, dim3((unsigned)((n + 255) / 256)), dim3(256), 0, dev.stream,
                    tab, T, half, inv);
}

cudaError_t rope_apply(int dtype, void* qkv, int64_t M, int64_t ld, int n_heads, int n_kv_heads,
                       int head_dim, int rotary_dim, const int32_t* pos, int T, const float2* tab,
                       const Dev& dev) {
  const int half = rotary_dim / 2;
  const int heads = n_heads + n_kv_heads;   // query heads then key heads are contiguous
  const int64_t n = M * heads * half;
  if (n <= 0) return cudaSuccess;
  const unsigned grid = (unsigned)((n + 255) / 256);
  if (dtype == kBF16)
    return launch_pdl(rope_apply_kernel<bf16>, dim3(grid), dim3(256), 0, dev.stream,
                      static_cast<bf16*>(qkv), M, ld, heads, head_dim, half, pos, T, tab);
  return launch_pdl(rope_apply_kernel<float>, dim3(grid), dim3(256), 0, dev.stream,
                    static_cast<float*>(qkv), M, ld, heads, head_dim, half, pos, T, tab);
}

cudaError_t router_f32(const float* x, int64_t n, int d, int h, const float* w1, const float* b1,
                       const float* w2, const float* b2, float* scores, const Dev& dev) {
  if (n <= 0) return cudaSuccess;
  return launch_pdl(router_f32_kernel, dim3(blocks_for(n, 8)), dim3(256), 0, dev.stream, x, n, d,
                    h, w1, b1, w2, b2, scores);
}

cudaError_t topk(const float* scores, int B, int T, int K, int32_t* idx, int32_t* rows,
                 const Dev& dev) {
  if (B <= 0 || K <= 0) return cudaSuccess;
  const size_t smem = (size_t)T * sizeof(uint32_t);
  static int attr_done[64] = {0};
  int device = 0;
  cudaGetDevice(&device);
  if (device < 64 && !attr_done[device]) {
    cudaError_t e = cudaFuncSetAttribute(topk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         kMaxTopkT * (int)sizeof(uint32_t));
    if (e != cudaSuccess) return e;
    attr_done[device] = 1;
  }
  return launch_pdl(topk_kernel, dim3(B), dim3(kTopkThreads), smem, dev.stream, scores, T, K, idx,
                    rows);
}

constexpr int kSelSmemMax = 2 * kMaxTopkT * 4 + 4 * 4096 * 4;   // keys, kept, fp32 params (d <= 4096)

template <typename T, bool RMS>
cudaError_t select_gather_norm_t(const float* scores, int B, int seq_len, int K, const void* x, int d,
                                 const void* g1, const void* b1, const void* g2, const void* b2,
                                 float eps, void* out1, void* out2, int32_t* idx, int32_t* rows,
                                 const Dev& dev) {
  const size_t smem = 4 * (size_t)d * sizeof(T) + (size_t)(seq_len + K) * 4;
  // Blocks per sequence: one row per warp when that keeps the grid within
  // about four blocks per SM (every block repeats the selection, so with
  // more rows each block takes several per warp).
  const int64_t per_block = std::max<int64_t>(kSelThreads / 32,
                                              ((int64_t)B * K + 4 * dev.num_sms - 1) / (4 * dev.num_sms));
  const int G = (int)std::max<int64_t>(1, (K + per_block - 1) / per_block);
  return with_nch<T>(d, [&](auto nch) -> cudaError_t {
    constexpr int NCH = decltype(nch)::value;
    static int attr_done[64] = {0};
    int device = 0;
    cudaGetDevice(&device);
    if (device < 64 && !attr_done[device]) {
      cudaError_t e = cudaFuncSetAttribute(select_gather_norm_kernel<T, RMS, NCH>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, kSelSmemMax);
      if (e != cudaSuccess) return e;
      attr_done[device] = 1;
    }
    return launch_pdl(select_gather_norm_kernel<T, RMS, NCH>, dim3(G, B), dim3(kSelThreads), smem,
                      dev.stream, scores, seq_len, K, static_cast<const T*>(x), d,
                      static_cast<const T*>(g1), static_cast<const T*>(b1),
                      static_cast<const T*>(g2), static_cast<const T*>(b2), eps,
                      static_cast<T*>(out1), static_cast<T*>(out2), idx, rows);
  });
}

cudaError_t select_gather_norm(int dtype, const float* scores, int B, int T, int K, const void* x,
                               int d, bool is_rms, const void* g1, const void* b1, const void* g2,
                               const void* b2, float eps, void* out1, void* out2, int32_t* idx,
                               int32_t* rows, const Dev& dev) {
  if (B <= 0 || K <= 0) return cudaSuccess;
  if (T > kMaxTopkT) return cudaErrorInvalidValue;
  if (dtype == kBF16)
    return is_rms ? select_gather_norm_t<bf16, true>(scores, B, T, K, x, d, g1, b1, g2, b2, eps,
                                                     out1, out2, idx, rows, dev)
                  : select_gather_norm_t<bf16, false>(scores, B, T, K, x, d, g1, b1, g2, b2, eps,
                                                      out1, out2, idx, rows, dev);
  return is_rms ? select_gather_norm_t<float, true>(scores, B, T, K, x, d, g1, b1, g2, b2, eps,
                                                    out1, out2, idx, rows, dev)
                : select_gather_norm_t<float, false>(scores, B, T, K, x, d, g1, b1, g2, b2, eps,
                                                     out1, out2, idx, rows, dev);
}

// Fixed block count for a given row count (independent of the device), so the
// fixed-order sums are reproducible everywhere.
int stats_partials_count(int64_t n_rows) {
  const int64_t want = (n_rows + (kStatThreads / 32) - 1) / (kStatThreads / 32);
  const int64_t cap = kStatMaxBlocks;
  return (int)(want < cap ? (want > 0 ? want : 1) : cap);
}

cudaError_t cos_stats(int dtype, const void* a, const void* b, int64_t n_rows, int d, int mode,
                      double* partials, double* acc, const Dev& dev) {
  if (n_rows <= 0) return cudaSuccess;
  const int nb = stats_partials_count(n_rows);
  cudaError_t e;
  if (dtype == kBF16)
    e = launch_pdl(cos_rows_kernel<bf16>, dim3(nb), dim3(kStatThreads), 0, dev.stream,
                   static_cast<const bf16*>(a), static_cast<const bf16*>(b), n_rows, d, mode, partials);
  else
    e = launch_pdl(cos_rows_kernel<float>, dim3(nb), dim3(kStatThreads), 0, dev.stream,
                   static_cast<const float*>(a), static_cast<const float*>(b), n_rows, d, mode,
                   partials);
  if (e != cudaSuccess) return e;
  return launch_pdl(cos_finish_kernel, dim3(1), dim3(256), 0, dev.stream, partials, nb, n_rows, mode,
                    acc);
}

cudaError_t cos_stats_chunks(const float4* parts, int64_t n_rows, int nch, int mode, double* partials,
                             double* acc, const Dev& dev) {
  if (n_rows <= 0) return cudaSuccess;
  const int nb = stats_partials_count(n_rows);
  cudaError_t e = launch_pdl(cos_chunks_kernel, dim3(nb), dim3(kStatThreads), 0, dev.stream, parts, n_rows, nch,
                             mode, partials);
  if (e != cudaSuccess) return e;
  return launch_pdl(cos_finish_kernel, dim3(1), dim3(256), 0, dev.stream, partials, nb, n_rows, mode, acc);
}

int stats_static_capacity() { return kStatMaxBlocks; }

// Same reduction as cos_stats, with the partial sums in g_stats_scratch. In
// host code g_stats_scratch names a host-side stand-in, not device memory, so
// its device address is looked up once per device (with that device current)
// and cached.
cudaError_t cos_stats_static(int dtype, const void* a, const void* b, int64_t n_rows, int d,
                             int mode, double* acc, const Dev& dev) {
  static std::mutex mu;
  static double* addr[64] = {nullptr};
  int device = 0;
  cudaError_t e = cudaGetDevice(&device);
  if (e != cudaSuccess) return e;
  if (device < 0 || device >= 64) return cudaErrorInvalidDevice;
  double* scratch = nullptr;
  {
    std::lock_guard<std::mutex> lk(mu);
    if (!addr[device]) {
      void* p = nullptr;
      e = cudaGetSymbolAddress(&p, g_stats_scratch);
      if (e != cudaSuccess) return e;
      addr[device] = static_cast<double*>(p);
    }
    scratch = addr[device];
  }
  if (stats_partials_count(n_rows) > kStatMaxBlocks) return cudaErrorInvalidValue;
  return cos_stats(dtype, a, b, n_rows, d, mode, scratch, acc, dev);
}

cudaError_t iota_positions(int32_t* idx, int B, int K, const Dev& dev) {
  const int64_t n = (int64_t)B * K;
  if (n <= 0) return cudaSuccess;
  return launch_pdl(iota_kernel, dim3((unsigned)((n + 255) / 256)), dim3(256), 0, dev.stream, idx, n,
                    K);
}

cudaError_t bounded_wait_selftest(int timeout_us, const Dev& dev) {
  bounded_wait_selftest_kernel<<<1, 32, 0, dev.stream>>>(dev.err,
                                                         (unsigned long long)timeout_us * 1000ull);
  return cudaGetLastError();
}

}  // namespace adadsf
