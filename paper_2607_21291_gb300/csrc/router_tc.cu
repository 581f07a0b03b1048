// Sec. 3.4: router scores of every token on the 5th-generation tensor cores
// (bf16): s = w2 . SiLU(W1 x + b1) + b2.
//
// H = X W1^T is a [B T, d] x [64, d]^T product (tcgen05, M = 128 tokens,
// N = 64 hidden units), cut into units of one 128-token tile x one 64-deep
// k-block. With at most one wave of tiles every CTA takes whole tiles (an
// exchange of partial tiles costs more than it saves); with more tiles than
// SMs the G CTAs take equal contiguous ranges of units, tile-major, so that
// no partial last wave leaves SMs idle, and a range may end inside a tile
// (the tile is then split along d). A tile whose
// units span several CTAs is finished by the last of them to get there: the
// others leave fp32 partial tiles in scratch (L2), and the finisher adds all
// partials in CTA order, so the sum does not depend on timing. No CTA ever
// waits for another: an atomic count per split tile only decides which CTA
// finishes it, and that CTA sets the count back to zero for the next launch.
// The counts live in the workspace's fixed synchronisation area (at the
// index of the tile's first CTA), so they stay valid whatever shapes other
// calls on the same workspace had. Ordering follows the usual release /
// acquire pattern: the group's partial-tile stores, a group barrier, then
// one thread's gpu-scope fence and atomic; the thread that sees the final
// count fences again before the group reads the partials.
//   warp 0      TMA: the X tile (128 x 64) and the W1 tile (64 x 64) of each unit
//   warp 1      TMEM (two 64-column accumulators); one thread issues the MMAs
//   warps 2-9   two per TMEM lane quarter, 32 hidden units each: partial
//               tiles and the score epilogue (a group of 256 threads on a
//               named barrier); on request also every token row's sum of
//               squares (the first RMSNorm's statistic), read from each
//               stage's token tile before the stage is freed, split tiles'
//               row sums travelling with their partial tiles
// Every barrier wait is bounded in time (device error word on give-up).
#include <algorithm>
#include <cstdlib>
#include <map>
#include <mutex>
#include <tuple>

#include "common.cuh"
#include "internal.h"

namespace adadsf {
namespace {

constexpr int kRM = 128;                 // tokens per tile = TMEM lanes
constexpr int kRN = 64;                  // router hidden units
constexpr int kRK = 64;                  // k-block depth: one 128-byte swizzled row of bf16
constexpr int kRStages = 6;
constexpr int kREpiWarps = 8;
constexpr int kREpiThreads = 32 * kREpiWarps;
constexpr int kRThreads = 64 + kREpiThreads;
constexpr int kRA = kRM * kRK * 2;       // X tile bytes
constexpr int kRB = kRN * kRK * 2;       // W1 tile bytes
constexpr int kRTile = kRM * kRN;        // floats of one partial tile
constexpr int kRMaxCtas = 160;           // partial-tile scratch slots: 2 per CTA
constexpr int kRBar = 1;                 // named barrier of the epilogue group

// shared-memory layout (offsets from the 1024-byte aligned base)
constexpr int kRRing = kRStages * (kRA + kRB);
constexpr int kROffBar = kRRing;
constexpr int kROffMisc = kROffBar + 256;
constexpr int kROffConst = kROffMisc + 128;
constexpr int kROffXchg = kROffConst + 2 * kRN * 4;
constexpr int kROffXsq = kROffXchg + 2 * kRM * 4;
constexpr int kRSmem = 1024 + kROffXsq + 2 * kRM * 4;   // with the alignment slack
// One CTA's partial of a split tile: the hidden-unit tile, then the sums of
// squares of the token rows over its k-blocks (one row of 128 per half).
constexpr int kRSlot = kRTile + 2 * kRM;
static_assert((2 * kRStages + 5) * 8 <= 256, "barrier area");
static_assert(kRMaxCtas * 4 <= (int)kSyncBytes, "tile counters");

struct RouterDev {
  int64_t rows;          // tokens (B T)
  int64_t U;             // units: n_tiles * nkb
  int nkb;               // k-blocks per tile (d / 64)
  int G;                 // CTAs
  const bf16* b1;
  const bf16* w2;
  const bf16* b2;
  float* scores;
  float* tsq;            // [rows] sum of squares of each token row of X, or null
  float* partials;       // [G][2][kRSlot]
  int* tile_cnt;         // [G]: split tile counted at its first CTA
  int* err;
  unsigned long long timeout_ns;
};

// First unit of CTA c (c = G: one past the last unit).
__device__ __forceinline__ int64_t unit_start(int64_t c, const RouterDev& p) { return c * p.U / p.G; }
// CTA whose range holds unit x: the largest c with unit_start(c) <= x.
__device__ __forceinline__ int unit_owner(int64_t x, const RouterDev& p) {
  return (int)(((x + 1) * p.G - 1) / p.U);
}
// Partial tiles: [hidden / 4][token][4] floats, so a warp moves 512
// contiguous bytes per 16-byte access.
__device__ __forceinline__ int partial_at(int row, int col) { return ((col >> 2) * kRM + row) * 4 + (col & 3); }

__device__ __forceinline__ float silu_r(float v) { return v * __fdividef(1.f, 1.f + __expf(fminf(-v, 80.f))); }

__device__ __forceinline__ void fence_gpu() { asm volatile("fence.acq_rel.gpu;" ::: "memory"); }

__global__ void __launch_bounds__(kRThreads, 1)
    router_tc_kernel(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmW,
                     const __grid_constant__ RouterDev p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const uint32_t sA = smem_u32(smem);
  const uint32_t sB = sA + kRStages * kRA;
  const uint32_t full0 = sA + kROffBar;
  const uint32_t empty0 = full0 + 8 * kRStages;
  const uint32_t tfull0 = empty0 + 8 * kRStages;
  const uint32_t tempty0 = tfull0 + 16;
  const uint32_t drain = tempty0 + 16;
  int* misc = reinterpret_cast<int*>(smem + kROffMisc);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(misc);
  volatile int* abort_flag = misc + 1;
  volatile int* last_flag = misc + 2;
  volatile int* ok_flags = misc + 4;   // [2][kREpiWarps]
  float* cst = reinterpret_cast<float*>(smem + kROffConst);   // b1[64], w2[64]
  float* xchg = reinterpret_cast<float*>(smem + kROffXchg);   // [2][128]
  float* xsq = reinterpret_cast<float*>(smem + kROffXsq);     // [2][128]

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int64_t u0 = unit_start(blockIdx.x, p);
  const int64_t u1 = unit_start((int64_t)blockIdx.x + 1, p);

  pdl_trigger();
  if (threadIdx.x == 0) {
    for (int s = 0; s < kRStages; ++s) {
      mbar_init(full0 + 8 * s, 1);
      // freed by the MMA commit and, with row statistics, each epilogue warp
      mbar_init(empty0 + 8 * s, p.tsq ? 1 + kREpiWarps : 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(tfull0 + 8 * a, 1);
      mbar_init(tempty0 + 8 * a, kREpiWarps);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_barrier_init();
    fence_proxy_async_smem();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmX);
    tma_prefetch_desc(&tmW);
  }
  if (warp == 1) tmem_alloc(smem_u32(tmem_slot), 2 * kRN);
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      const int64_t n = u1 - u0;
      const int pre = (int)(n < kRStages ? n : kRStages);
      // W1 does not depend on the previous kernel: the first stages' weight
      // tiles are requested before waiting for it
      for (int i = 0; i < pre; ++i) {
        const int kb = (int)((u0 + i) % p.nkb);
        mbar_arrive_expect_tx(full0 + 8 * i, kRA + kRB);
        tma_load_2d(sB + i * kRB, &tmW, kb * kRK, 0, full0 + 8 * i);
      }
      pdl_wait();
      int stage = 0;
      uint32_t phase = 0;
      int64_t issued = 0;
      for (int64_t u = u0; u < u1; ++u) {
        const int64_t tile = u / p.nkb;
        const int kc = (int)(u - tile * p.nkb) * kRK;
        const uint32_t fb = full0 + 8 * stage;
        if (issued >= pre) {
          if (!mbar_wait_bounded(empty0 + 8 * stage, phase ^ 1, abort_flag, p.err, p.timeout_ns)) break;
          mbar_arrive_expect_tx(fb, kRA + kRB);
          tma_load_2d(sB + stage * kRB, &tmW, kc, 0, fb);
        }
        tma_load_2d(sA + stage * kRA, &tmX, kc, (int)(tile * kRM), fb);
        ++issued;
        if (++stage == kRStages) { stage = 0; phase ^= 1; }
      }
      // Drain: wait until the last copy issued into each stage has landed.
      for (int s = 0; s < kRStages; ++s) {
        if (issued <= s) break;
        const int64_t last = s + ((issued - 1 - s) / kRStages) * kRStages;
        mbar_wait_drain(full0 + 8 * s, (uint32_t)((last / kRStages) & 1), p.timeout_ns);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(kRM, kRN);
      int stage = 0;
      uint32_t phase = 0;
      int it = 0;
      bool ok = true;
      int64_t u = u0;
      while (u < u1 && ok) {
        const int64_t tile = u / p.nkb;
        const int64_t uend = min(u1, (tile + 1) * p.nkb);
        const int acc = it & 1;
        if (!mbar_wait_bounded(tempty0 + 8 * acc, ((it >> 1) & 1) ^ 1, abort_flag, p.err, p.timeout_ns)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * kRN;
        const int64_t useg = u;
        for (; u < uend; ++u) {
          if (!mbar_wait_bounded(full0 + 8 * stage, phase, abort_flag, p.err, p.timeout_ns)) {
            ok = false;
            break;
          }
          tc_fence_after();
#pragma unroll
          for (int k = 0; k < kRK / 16; ++k)
            tc_mma_f16(d_tmem, smem_desc_sw128(sA + stage * kRA + k * 32),
                       smem_desc_sw128(sB + stage * kRB + k * 32), idesc, (u > useg || k > 0) ? 1u : 0u);
          tc_commit(empty0 + 8 * stage);   // stage free once these MMAs have read it
          if (++stage == kRStages) { stage = 0; phase ^= 1; }
        }
        if (!ok) break;
        tc_commit(tfull0 + 8 * acc);       // accumulator ready
        ++it;
      }
      tc_commit(drain);
      mbar_wait_drain(drain, 0, p.timeout_ns);
    }
  } else {
    // ------------------------------------------------------------ epilogue (warps 2..9)
    const int ew = warp - 2;
    const int quarter = warp & 3;           // TMEM lanes 32 quarter .. +31
    const int half = ew >> 2;               // hidden units [32 half, 32 half + 32)
    const int r = quarter * 32 + lane;      // token in the tile
    const int etid = threadIdx.x - 64;
    const auto esync = [] { named_bar_sync(kRBar, kREpiThreads); };
    if (etid < kRN) {   // weights: independent of the previous kernel
      cst[etid] = __bfloat162float(p.b1[etid]);
      cst[kRN + etid] = __bfloat162float(p.w2[etid]);
    }
    const float b2 = __bfloat162float(p.b2[0]);
    pdl_wait();
    esync();
    int it = 0, seg = 0;
    int64_t u = u0;
    // row statistics: the ring stage and phase of the next unit
    int sstage = 0;
    uint32_t sphase = 0;
    bool sok = true;
    while (u < u1) {
      const int64_t tile = u / p.nkb;
      const int64_t tstart = tile * p.nkb, tend = tstart + p.nkb;
      const int64_t uend = min(u1, tend);
      const bool whole = u == tstart && uend == tend;
      const int acc = it & 1;
      // Sum of squares of token row r over this segment's k-blocks: the
      // thread reads its half of the row's 128-byte swizzled line (16-byte
      // chunk c sits at c ^ (r % 8)) from each stage, then frees the stage
      // with its warp.
      float sq0 = 0.f, sq1 = 0.f;
      if (p.tsq) {
        for (int64_t v = u; v < uend; ++v) {
          if (sok) {
            int sw = 1;
            if (lane == 0) sw = mbar_wait_bounded(full0 + 8 * sstage, sphase, abort_flag, p.err, p.timeout_ns);
            sok = __shfl_sync(0xffffffffu, sw, 0) != 0;
            __syncwarp();   // the other lanes' reads follow lane 0's observation of the stage
          }
          if (sok) {
            const uint4* line = reinterpret_cast<const uint4*>(smem + sstage * kRA + r * 128);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              const uint4 q = line[(4 * half + i) ^ (r & 7)];
              const uint32_t wv[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
              for (int j = 0; j < 4; ++j) {
                const float lo = __uint_as_float(wv[j] << 16), hi = __uint_as_float(wv[j] & 0xffff0000u);
                sq0 = fmaf(lo, lo, sq0);
                sq1 = fmaf(hi, hi, sq1);
              }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(empty0 + 8 * sstage);
          }
          if (++sstage == kRStages) { sstage = 0; sphase ^= 1; }
        }
      }
      const float sq = sq0 + sq1;
      int w = 1;
      if (lane == 0) w = mbar_wait_bounded(tfull0 + 8 * acc, (it >> 1) & 1, abort_flag, p.err, p.timeout_ns);
      w = __shfl_sync(0xffffffffu, w, 0);
      // the group leaves together: every warp's wait result is shared first
      if (lane == 0) ok_flags[acc * kREpiWarps + ew] = w;
      esync();
      bool all_ok = true;
#pragma unroll
      for (int i = 0; i < kREpiWarps; ++i) all_ok = all_ok && ok_flags[acc * kREpiWarps + i] != 0;
      if (!all_ok) break;
      tc_fence_after();
      uint32_t raw[32];
      tmem_ld32(tmem_base + ((uint32_t)(quarter * 32) << 16) + acc * kRN + half * 32, raw);
      tmem_ld_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(tempty0 + 8 * acc);   // accumulator free for the next segment
      float v[32];
#pragma unroll
      for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(raw[j]);
      bool fin = whole;
      if (!whole) {
        // partial tile: slot 0 holds a CTA's first segment, slot 1 its last
        float* mine = p.partials + ((size_t)blockIdx.x * 2 + (seg == 0 ? 0 : 1)) * kRSlot;
#pragma unroll
        for (int j = 0; j < 8; ++j)
          __stcg(reinterpret_cast<float4*>(mine + partial_at(r, half * 32 + 4 * j)),
                 make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]));
        if (p.tsq) __stcg(mine + kRTile + half * kRM + r, sq);
        esync();
        const int c_lo = unit_owner(tstart, p), c_hi = unit_owner(tend - 1, p);
        if (etid == 0) {
          fence_gpu();   // release the group's partial tile
          const int old = atomicAdd(p.tile_cnt + c_lo, 1);
          const int last = old == c_hi - c_lo;
          if (last) {
            atomicExch(p.tile_cnt + c_lo, 0);
            fence_gpu();   // acquire the other CTAs' partial tiles
          }
          *last_flag = last;
        }
        esync();
        fin = *last_flag != 0;
        if (fin) {
          float s[32];
#pragma unroll
          for (int j = 0; j < 32; ++j) s[j] = 0.f;
          for (int c = c_lo; c <= c_hi; ++c) {
            if (c == (int)blockIdx.x) {
#pragma unroll
              for (int j = 0; j < 32; ++j) s[j] += v[j];
            } else {
              const int slot = unit_start(c, p) / p.nkb == tile ? 0 : 1;
              const float* src = p.partials + ((size_t)c * 2 + slot) * kRSlot;
#pragma unroll
              for (int j = 0; j < 8; ++j) {
                const float4 f = __ldcg(reinterpret_cast<const float4*>(src + partial_at(r, half * 32 + 4 * j)));
                s[4 * j] += f.x;
                s[4 * j + 1] += f.y;
                s[4 * j + 2] += f.z;
                s[4 * j + 3] += f.w;
              }
            }
          }
#pragma unroll
          for (int j = 0; j < 32; ++j) v[j] = s[j];
        }
      }
      if (fin) {
        // s = w2 . SiLU(h + b1) + b2 over both halves of the hidden units
        float part[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int j = 0; j < 32; ++j)
          part[j & 3] += cst[kRN + half * 32 + j] * silu_r(v[j] + cst[half * 32 + j]);
        const float mine = (part[0] + part[1]) + (part[2] + part[3]);
        float* xb = xchg + acc * kRM;
        if (half == 1) {
          xb[r] = mine;
          if (p.tsq && whole) xsq[acc * kRM + r] = sq;
        }
        esync();
        const int64_t row = tile * kRM + r;
        if (half == 0 && row < p.rows) {
          p.scores[row] = (mine + xb[r]) + b2;
          if (p.tsq) {
            float t = 0.f;
            if (whole) {
              t = sq + xsq[acc * kRM + r];
            } else {
              // every contributing CTA's two half-row sums, in CTA order
              for (int c = unit_owner(tstart, p); c <= unit_owner(tend - 1, p); ++c) {
                const int slot = unit_start(c, p) / p.nkb == tile ? 0 : 1;
                const float* src = p.partials + ((size_t)c * 2 + slot) * kRSlot + kRTile;
                t += __ldcg(src + r) + __ldcg(src + kRM + r);
              }
            }
            p.tsq[row] = t;
          }
        }
      }
      u = uend;
      ++seg;
      ++it;
    }
  }

  // Reconverge each warp first: in the producer and MMA warps only lane 0
  // ran the role loop, and the block barrier counts whole warps.
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, 2 * kRN);
  }
}

// ---------------------------------------------------------------- host side
int64_t owner_host(int64_t x, int64_t U, int G) { return ((x + 1) * G - 1) / U; }

// Cost, in k-block units (~0.33 us each on GB300), of G CTAs over n_tiles x
// nkb units: the longest range, plus the partial-tile exchange of the most
// split tile (measured ~4.5 us for a two-way split: the partial-tile stores,
// two gpu-scope fences, the atomic and the partial-tile loads in series).
double router_cost(int64_t n_tiles, int nkb, int G) {
  const int64_t U = n_tiles * nkb;
  const int64_t per = (U + G - 1) / G;
  int64_t contrib = 1;
  for (int64_t t = 0; t < n_tiles; ++t) {
    const int64_t c = owner_host((t + 1) * nkb - 1, U, G) - owner_host(t * nkb, U, G) + 1;
    contrib = std::max(contrib, c);
  }
  return (double)per + (contrib > 1 ? 14.0 + 2.0 * (double)(contrib - 2) : 0.0);
}

// Tuning override: ADADSF_ROUTER_SPLIT=s (s >= 1) splits every tile s ways
// (capped by the SMs and the scratch slots); unset or 0 chooses by the cost
// model.
int router_split_override() {
  static int v = -1;
  if (v < 0) {
    const char* e = getenv("ADADSF_ROUTER_SPLIT");
    v = e ? atoi(e) : 0;
    if (v < 0) v = 0;
  }
  return v;
}

// CTAs for n_tiles x nkb units: whole tiles per CTA without scratch, else
// the cheapest of n_tiles x s (s-way split of every tile) and one range per
// SM (stream order), capped by the scratch slots. Cached per shape.
int router_ctas(int64_t n_tiles, int nkb, int sms, bool split) {
  if (!split) return (int)n_tiles;
  if (const int s = router_split_override()) {
    if (s == 1) return (int)n_tiles;
    return (int)std::min<int64_t>(std::min<int64_t>(n_tiles * s, std::min(sms, kRMaxCtas)), n_tiles * nkb);
  }
  static std::mutex mu;
  static std::map<std::tuple<int64_t, int, int>, int> cache;
  const auto key = std::make_tuple(n_tiles, nkb, sms);
  std::lock_guard<std::mutex> lock(mu);
  auto f = cache.find(key);
  if (f != cache.end()) return f->second;
  const int cap = std::min(sms, kRMaxCtas);
  const int64_t U = n_tiles * nkb;
  int best = (int)std::min<int64_t>(n_tiles, cap);
  double best_cost = n_tiles > cap ? 1e30 : router_cost(n_tiles, nkb, best);
  if (n_tiles > cap) {
    // whole tiles in waves vs one range per SM
    best = (int)n_tiles;
    best_cost = (double)((n_tiles + sms - 1) / sms) * nkb;
  }
  for (int s = 1; s <= nkb; ++s) {
    const int G = (int)std::min<int64_t>(std::min<int64_t>(n_tiles * s, cap), U);
    const double c = router_cost(n_tiles, nkb, G);
    if (c < best_cost) {
      best_cost = c;
      best = G;
    }
    if (n_tiles * s >= cap) break;
  }
  cache[key] = best;
  return best;
}

}  // namespace

size_t router_partial_bytes() { return (size_t)kRMaxCtas * 2 * kRSlot * 4; }

cudaError_t router_tc(const void* x, int64_t rows, int d, const void* w1, const void* b1, const void* w2,
                      const void* b2, float* scores, float* tsq, int* sync, float* partials, const Dev& dev) {
  if (rows <= 0) return cudaSuccess;
  if (d % kRK != 0 || d <= 0) return cudaErrorInvalidValue;
  const int64_t n_tiles = (rows + kRM - 1) / kRM;
  const int nkb = d / kRK;
  RouterDev p{};
  p.rows = rows;
  p.nkb = nkb;
  p.U = n_tiles * nkb;
  p.G = router_ctas(n_tiles, nkb, dev.num_sms, sync && partials);
  p.b1 = static_cast<const bf16*>(b1);
  p.w2 = static_cast<const bf16*>(w2);
  p.b2 = static_cast<const bf16*>(b2);
  p.scores = scores;
  p.tsq = tsq;
  p.tile_cnt = sync;
  p.partials = partials;
  p.err = dev.err;
  p.timeout_ns = kWaitTimeoutNs;
  CUtensorMap tx, tw;
  if (!make_tmap_bf16(&tx, x, (uint64_t)rows, (uint64_t)d, (uint64_t)d, kRK, kRM) ||
      !make_tmap_bf16(&tw, w1, (uint64_t)kRN, (uint64_t)d, (uint64_t)d, kRK, kRN))
    return cudaErrorInvalidValue;
  static std::once_flag attr_once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(attr_once, [] {
    attr_err = cudaFuncSetAttribute(router_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kRSmem);
  });
  if (attr_err != cudaSuccess) return attr_err;
  return launch_pdl(router_tc_kernel, dim3(p.G), dim3(kRThreads), kRSmem, dev.stream, tx, tw, p);
}

}  // namespace adadsf
