// Eq. 1 among the kept tokens on the 5th-generation tensor cores (bf16).
//
// Work items are (pair of 128-query blocks, query head, sequence): the two
// query tiles share every K / V tile loaded, which halves the K / V traffic
// per flop, and their softmax work alternates with the other tile's matrix
// products. When pairs would leave SMs idle (few, short sequences), one
// query block per item instead. The kernel is persistent: one CTA per SM
// walks its share of the items (longest causal rows first), the K / V rings
// and every barrier phase running on across items, so one item's output
// epilogue overlaps the next item's Q load and first scores, and the CTA's
// set-up (barriers, TMEM) is paid once. Keys arrive in blocks of 128; attention is causal in
// packed order (kept positions ascend, so this is the original causal mask
// restricted to the kept set, Sec. 3.4).
//   warp 0     TMA, lane 0: both Q tiles once, then the K tile of each key
//              block into a ring released once both tiles' S of that block
//              are done; lane 1: the V^T tile of each key block into a ring
//              released after both tiles' P V (128-byte swizzled, K-major
//              operands). The two lanes run their loops independently.
//   warp 1     allocates TMEM; one thread issues, per tile t, S_t = Q_t K^T
//              (tcgen05.mma, M = 128, N = 128) into TMEM S_t and, once the
//              tile's softmax warps have written P_t over S_t (bf16 pairs),
//              O_t += P_t V with P_t read from TMEM as the A operand. The
//              order S_0(j) S_1(j) P_0V(j) S_0(j+1) P_1V(j) S_1(j+1) ... keeps
//              the tensor pipe busy with one tile while the other's softmax
//              runs; a tile's next S is issued after its P V, and the
//              tensor-core pipe runs one thread's operations in order.
//   warps 2-9  softmax of tile 0, warps 10-17 of tile 1: two warps per TMEM
//              lane quarter, one query row and 64 of the 128 key columns per
//              thread (the pair exchanges row maxima and sums through shared
//              memory on a named barrier): read S once, mask (diagonal block
//              only), online softmax in fp32 (exp2 with a row maximum held at
//              most 2^8 below the true one, so O is rescaled only when the
//              maximum grows by more than that; paired fp32 arithmetic and
//              three-input maxima keep the instruction count down), write P
//              as bf16 pairs over
//              the first 32 of its own 64 S columns (so neither warp of the
//              pair overwrites scores the other has yet to read), and at the
//              end O / l -> global.
//              When S_t(j) is complete, P_t V of block j-1 is too (same pipe,
//              issued earlier), so the rescale of O_t and the overwrite of
//              P_t need no other wait.
// V enters as V^T (features x keys per key-value head), written by the QKV
// projection's epilogue.
// Every barrier wait is bounded in time (device error word on give-up).
#include <cuda.h>

#include "common.cuh"
#include "internal.h"

namespace adadsf {
namespace {

constexpr int kQB = 128;            // queries per tile = TMEM lanes
constexpr int kKB = 128;            // keys per block
constexpr int kSoftWarps = 16;      // eight per tile, two per TMEM lane quarter
constexpr int kAttnThreads = 32 * (2 + kSoftWarps);
constexpr float kRescaleLog2 = 8.f; // O rescaled only when the row max grows by > 2^8

template <int HD>
struct AttnCfg {
  static constexpr int KST = HD == 64 ? 4 : 3;     // K ring stages
  static constexpr int VST = HD == 64 ? 4 : 2;     // V^T ring stages
  static constexpr int HS = HD / 64;               // 64-feature slabs of a head row
  static constexpr int SLAB = kQB * 128;           // one 128-row x 128-byte slab
  static constexpr int Q_BYTES = HS * SLAB;        // one query tile
  static constexpr int K_BYTES = HS * SLAB;
  static constexpr int V_SLAB = HD * 128;          // HD feature rows x 64 keys
  static constexpr int V_BYTES = 2 * V_SLAB;       // 128 keys
  static constexpr int DATA = 2 * Q_BYTES + KST * K_BYTES + VST * V_BYTES;
  static constexpr int NBARS = 1 + 2 * KST + 2 * VST + 10;
  // barriers, TMEM address, abort flag; then the softmax pairs' exchange
  // area: [tile][quarter][half][lane] floats
  static constexpr int XCHG = 2 * 4 * 2 * 32 * 4;
  static constexpr int TAIL = 256 + XCHG;
  // Room left for aligning the dynamic base to 1024 bytes (the kernel checks
  // its actual misalignment); padded so that one CTA holds an SM (TMEM is
  // allocated in full).
  static constexpr int SLACK = (232448 - DATA - TAIL) < 1024 ? (232448 - DATA - TAIL) : 1024;
  static constexpr int SMEM_RAW = DATA + TAIL + SLACK;
  static constexpr int SMEM = SMEM_RAW > 120 * 1024 ? SMEM_RAW : 120 * 1024;
  static_assert(SLACK >= 256, "shared memory");
  static_assert(NBARS * 8 + 8 <= TAIL, "barrier area");
  // TMEM: S_0 (P_0 over its first 64 columns) at 0, S_1 at 128, O_0 at 256,
  // O_1 at 256 + HD
  static constexpr uint32_t TS = 0, TO = 256;
  static_assert(TO + 2 * HD <= 512, "TMEM columns");
};

// 2^x on the SFU (ex2.approx.ftz.f32: relative error ~2^-22, flushes
// denormal results; P is rounded to bf16 afterwards).
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// max(a, b, c) in one instruction.
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

struct AttnDev {
  int K;                 // kept tokens per sequence
  int pair;              // 1: two query blocks per work item, 0: one
  int B, Hq, Hkv, q_dim;
  float scale_log2;      // log2(e) / sqrt(hd)
  bf16* out;
  int64_t ld_out;
  int* err;
  unsigned long long timeout_ns;
};

// Work item w of the persistent schedule: query head h, sequence b and
// query-block group z (z = 0 holds each (head, sequence)'s longest causal
// rows). Items are numbered h fastest, then b, then z, so the longest rows of
// every head and sequence come first; CTA c takes items c, c + G, c + 2G, ...
struct AttnItem {
  int h, b, qb0, two, n_kv, g, row0;
};
__device__ __forceinline__ AttnItem attn_item(const AttnDev& p, int w, int nqb) {
  AttnItem it;
  it.h = w % p.Hq;
  it.b = (w / p.Hq) % p.B;
  const int z = w / (p.Hq * p.B);
  it.qb0 = p.pair ? 2 * ((nqb + 1) / 2 - 1 - z) : nqb - 1 - z;
  it.two = (p.pair && it.qb0 + 1 < nqb) ? 1 : 0;   // tile 1 holds query block qb0 + 1
  it.n_kv = it.two ? it.qb0 + 2 : it.qb0 + 1;        // tile 0 takes blocks 0..qb0, tile 1 all
  it.g = it.h / (p.Hq / p.Hkv);
  it.row0 = it.b * p.K;
  return it;
}

template <int HD>
__global__ void __launch_bounds__(kAttnThreads, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tmQK, const __grid_constant__ CUtensorMap tmVt,
                   const AttnDev p) {
  using C = AttnCfg<HD>;
  constexpr int KST = C::KST, VST = C::VST;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  if (smem - smem_raw > C::SLACK) {   // the layout would not fit: report and touch nothing
    if (threadIdx.x == 0) set_device_error(p.err, DEVERR_TIMEOUT);
    return;
  }
  const uint32_t sQ = smem_u32(smem);                  // [2] query tiles
  const uint32_t sK0 = sQ + 2 * C::Q_BYTES;
  const uint32_t sV0 = sK0 + KST * C::K_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::DATA);
  const uint32_t b0 = smem_u32(bars);
  const uint32_t q_full = b0;
  const uint32_t k_full0 = b0 + 8;                 // [KST]
  const uint32_t k_empty0 = k_full0 + 8 * KST;     // [KST]
  const uint32_t v_full0 = k_empty0 + 8 * KST;     // [VST]
  const uint32_t v_empty0 = v_full0 + 8 * VST;     // [VST]
  const uint32_t s_full0 = v_empty0 + 8 * VST;     // [2] per tile: S_t of the block done
  const uint32_t p_full0 = s_full0 + 16;           // [2] per tile: P_t written (8 warps)
  const uint32_t o_done0 = p_full0 + 16;           // [2] per tile: P_t V of the block done
  const uint32_t drain = o_done0 + 16;
  const uint32_t q_empty = drain + 8;              // the item's S products have read Q
  const uint32_t o_free0 = q_empty + 8;            // [2] per tile: O_t read out (8 warps)
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + C::NBARS);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  // softmax pairs' exchange: [tile][quarter][half][lane]
  volatile float* xchg = reinterpret_cast<volatile float*>(smem + C::DATA + 256);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int nqb = (p.K + kQB - 1) / kQB;
  const int n_items = p.Hq * p.B * (p.pair ? (nqb + 1) / 2 : nqb);

  pdl_trigger();
  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    mbar_init(q_empty, 1);
    for (int i = 0; i < KST; ++i) {
      mbar_init(k_full0 + 8 * i, 1);
      mbar_init(k_empty0 + 8 * i, 1);
    }
    for (int i = 0; i < VST; ++i) {
      mbar_init(v_full0 + 8 * i, 1);
      mbar_init(v_empty0 + 8 * i, 1);
    }
    for (int t = 0; t < 2; ++t) {
      mbar_init(s_full0 + 8 * t, 1);
      mbar_init(p_full0 + 8 * t, 8);
      mbar_init(o_done0 + 8 * t, 1);
      mbar_init(o_free0 + 8 * t, 8);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_barrier_init();
    fence_proxy_async_smem();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmQK);
    tma_prefetch_desc(&tmVt);
  }
  if (warp == 1) tmem_alloc(smem_u32(tmem_slot), 512);
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producers
    // lane 0: each item's Q tiles (once the previous item's scores are done
    // with Q), then its K blocks into the ring; lane 1: the V^T ring. Ring
    // positions run on across items.
    if (lane < 2) {
      const bool kprod = lane == 0;
      const int NST = kprod ? KST : VST;
      pdl_wait();
      const uint32_t full0 = kprod ? k_full0 : v_full0;
      const uint32_t empty0 = kprod ? k_empty0 : v_empty0;
      int issued = 0;   // ring position (copies issued)
      int it = 0;       // items of this CTA
      bool ok = true;
      for (int w = blockIdx.x; ok && w < n_items; w += gridDim.x, ++it) {
        const AttnItem I = attn_item(p, w, nqb);
        if (kprod) {
          if (it > 0 && !mbar_wait_bounded(q_empty, (it - 1) & 1, abort_flag, p.err, p.timeout_ns)) break;
          mbar_arrive_expect_tx(q_full, (I.two ? 2 : 1) * C::Q_BYTES);
          for (int t = 0; t < (I.two ? 2 : 1); ++t)
            for (int s = 0; s < C::HS; ++s)
              tma_load_2d(sQ + t * C::Q_BYTES + s * C::SLAB, &tmQK, I.h * HD + s * 64,
                          I.row0 + (I.qb0 + t) * kQB, q_full);
        }
        for (int j = 0; j < I.n_kv; ++j) {
          const int st = issued % NST;
          if (!mbar_wait_bounded(empty0 + 8 * st, ((issued / NST) & 1) ^ 1, abort_flag, p.err, p.timeout_ns)) {
            ok = false;
            break;
          }
          const uint32_t fb = full0 + 8 * st;
          if (kprod) {
            mbar_arrive_expect_tx(fb, C::K_BYTES);
            for (int s = 0; s < C::HS; ++s)
              tma_load_2d(sK0 + st * C::K_BYTES + s * C::SLAB, &tmQK, p.q_dim + I.g * HD + s * 64,
                          I.row0 + j * kKB, fb);
          } else {
            mbar_arrive_expect_tx(fb, C::V_BYTES);
            for (int ks = 0; ks < 2; ++ks)
              tma_load_2d(sV0 + st * C::V_BYTES + ks * C::V_SLAB, &tmVt, j * kKB + ks * 64,
                          (I.b * p.Hkv + I.g) * HD, fb);
          }
          ++issued;
        }
      }
      // drain: the copies issued last into each stage (and the last Q) have landed
      if (kprod && it > 0) mbar_wait_drain(q_full, (it - 1) & 1, p.timeout_ns);
      for (int st = 0; st < NST && st < issued; ++st) {
        const int last = st + ((issued - 1 - st) / NST) * NST;
        mbar_wait_drain(full0 + 8 * st, (uint32_t)((last / NST) & 1), p.timeout_ns);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc_s = idesc_bf16_f32(kQB, kKB);
      constexpr uint32_t idesc_o = idesc_bf16_f32(kQB, HD);
      // S_t(j) = Q_t K(j)^T into TMEM S_t, K block in ring slot kslot
      auto issue_s = [&](int t, int kslot) {
        const uint32_t kst = sK0 + kslot * C::K_BYTES;
        const uint32_t qt = sQ + t * C::Q_BYTES;
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk) {
          const uint32_t off = (kk >> 2) * C::SLAB + (kk & 3) * 32;
          tc_mma_f16(tmem_base + C::TS + t * kKB, smem_desc_sw128(qt + off), smem_desc_sw128(kst + off),
                     idesc_s, kk > 0 ? 1u : 0u);
        }
        tc_commit(s_full0 + 8 * t);
      };
      // O_t (+)= P_t V, P_t read from TMEM, V^T block in ring slot vslot
      auto issue_pv = [&](int t, int vslot, bool acc) {
        const uint32_t vst = sV0 + vslot * C::V_BYTES;
#pragma unroll
        for (int kk = 0; kk < kKB / 16; ++kk)   // keys 16 kk.. of P_t: columns 64 (kk / 4) + 8 (kk % 4)
          tc_mma_f16_ta(tmem_base + C::TO + t * HD, tmem_base + C::TS + t * kKB + (kk >> 2) * 64 + (kk & 3) * 8,
                        smem_desc_sw128(vst + (kk >> 2) * C::V_SLAB + (kk & 3) * 32), idesc_o,
                        (acc || kk > 0) ? 1u : 0u);
        tc_commit(o_done0 + 8 * t);
      };
      auto wait = [&](uint32_t bar, uint32_t parity) {
        return mbar_wait_bounded(bar, parity, abort_flag, p.err, p.timeout_ns);
      };
      int kc = 0, vc = 0;          // ring positions of the K and V^T blocks
      int pc[2] = {0, 0};          // P_t blocks consumed per tile
      int oc[2] = {0, 0};          // items finished per tile (their O read out)
      bool ok = true;
      int it = 0;
      for (int w = blockIdx.x; ok && w < n_items; w += gridDim.x, ++it) {
        const AttnItem I = attn_item(p, w, nqb);
        const int last0 = I.qb0;   // tile 0's last key block
        ok = wait(q_full, it & 1) && wait(k_full0 + 8 * (kc % KST), (kc / KST) & 1);
        if (!ok) break;
        tc_fence_after();
        // S_t(0) may overwrite the previous item's P_t: its P V was issued
        // before, and one thread's tcgen05 operations run in order
        issue_s(0, kc % KST);
        if (I.two) issue_s(1, kc % KST);
        tc_commit(k_empty0 + 8 * (kc % KST));
        for (int j = 0; j < I.n_kv; ++j) {
          const bool has0 = j <= last0;
          const bool next = j + 1 < I.n_kv;
          const int vslot = vc % VST;
          const int knext = (kc + 1) % KST;
          if (!wait(v_full0 + 8 * vslot, (vc / VST) & 1)) { ok = false; break; }
          if (has0) {
            if (!wait(p_full0, pc[0] & 1)) { ok = false; break; }
            ++pc[0];
            // the first P V of an item overwrites O_0: the previous item's
            // epilogue must have read it out
            if (j == 0 && oc[0] > 0 && !wait(o_free0, (oc[0] - 1) & 1)) { ok = false; break; }
            tc_fence_after();
            issue_pv(0, vslot, j > 0);
          }
          if (next && !wait(k_full0 + 8 * knext, ((kc + 1) / KST) & 1)) { ok = false; break; }
          tc_fence_after();
          if (next && j + 1 <= last0) issue_s(0, knext);
          if (I.two) {
            if (!wait(p_full0 + 8, pc[1] & 1)) { ok = false; break; }
            ++pc[1];
            if (j == 0 && oc[1] > 0 && !wait(o_free0 + 8, (oc[1] - 1) & 1)) { ok = false; break; }
            tc_fence_after();
            issue_pv(1, vslot, j > 0);
            if (next) issue_s(1, knext);
          }
          tc_commit(v_empty0 + 8 * vslot);            // V(j) read by both tiles
          ++vc;
          if (next) {
            tc_commit(k_empty0 + 8 * knext);          // K(j+1) read by both tiles
            ++kc;
          }
        }
        if (!ok) break;
        ++kc;                                  // past the item's last K block
        for (int t = 0; t < 2; ++t)
          if (t == 0 || I.two) ++oc[t];
        tc_commit(q_empty);                    // the item's scores are done with Q
      }
      tc_commit(drain);
      mbar_wait_drain(drain, 0, p.timeout_ns);
    }
  } else {
    // ------------------------------------------------------------ softmax (warps 2..17)
    pdl_wait();
    const int t = (warp - 2) >> 3;                 // tile
    const int half = ((warp - 2) >> 2) & 1;        // key columns [64 half, 64 half + 64)
    const int quarter = warp & 3;
    const int r = quarter * 32 + lane;             // query row in the tile = TMEM lane
    const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;
    const uint32_t tS = tmem_base + C::TS + t * kKB + lane_off;
    const uint32_t tO = tmem_base + C::TO + t * HD + lane_off + half * (HD / 2);
    const int bar_id = 1 + t * 4 + quarter;        // named barrier of the warp pair
    volatile float* xq = xchg + (t * 4 + quarter) * 64;
    // partner's value (same rows, other half of the columns); the second
    // barrier lets the next exchange reuse the slots
    auto exchange = [&](float mine) {
      xq[half * 32 + lane] = mine;
      named_bar_sync(bar_id, 64);
      const float theirs = xq[(half ^ 1) * 32 + lane];
      named_bar_sync(bar_id, 64);
      return theirs;
    };
    int sc = 0;    // S_t blocks consumed (the s_full phase)
    int pvc = 0;   // P_t V products of earlier items (the o_done phase)
    bool ok = true;
    for (int wi = blockIdx.x; ok && wi < n_items; wi += gridDim.x) {
    const AttnItem I = attn_item(p, wi, nqb);
    if (t == 1 && !I.two) continue;                // this item has one query tile
    const int qbt = I.qb0 + t;
    const int qi = qbt * kQB + r;                  // query index in the sequence
    float m_used = -INFINITY, l = 0.f;
    for (int j = 0; ok && j <= qbt; ++j) {
      int w = 0;
      if (lane == 0) w = mbar_wait_bounded(s_full0 + 8 * t, sc & 1, abort_flag, p.err, p.timeout_ns);
      ++sc;
      w = __shfl_sync(0xffffffffu, w, 0);
      tc_fence_after();
      const uint32_t tSh = tS + half * 64;         // this half's 64 score columns
      // keys above lim (relative to this half) are masked: diagonal block only
      const bool diag = j == qbt;
      const int lim = diag ? qi - j * kKB - half * 64 : kKB;
      float mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
      if (w) {
        uint32_t u[64];
        tmem_ld32(tSh, u);
        tmem_ld32(tSh + 32, u + 32);
        tmem_ld_wait();
        if (diag) {
#pragma unroll
          for (int i = 0; i < 64; ++i) mx[i & 3] = fmaxf(mx[i & 3], (i <= lim) ? __uint_as_float(u[i]) : -INFINITY);
        } else {
#pragma unroll
          for (int i = 0; i < 64; i += 2)
            mx[(i >> 1) & 3] = fmax3(mx[(i >> 1) & 3], __uint_as_float(u[i]), __uint_as_float(u[i + 1]));
        }
      }
      // a wait that gave up travels as NaN, so the pair leaves together (the
      // exchange is a barrier of both warps)
      const float part = w ? fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])) : NAN;
      const float other = exchange(part);
      if (part != part || other != other) { ok = false; break; }
      const float bmax = fmaxf(part, other) * p.scale_log2;
      bool need = false;
      if (j == 0) m_used = bmax;
      else need = bmax > m_used + kRescaleLog2;
      if (__any_sync(0xffffffffu, need)) {
        // O_t is stable: P_t V of block j - 1 completed before S_t(j)
        const float alpha = need ? ex2_approx(m_used - bmax) : 1.f;
        if (need) {
          l *= alpha;
          m_used = bmax;
        }
#pragma unroll 1
        for (int c = 0; c < HD / 64; ++c) {
          uint32_t o[32];
          tmem_ld32(tO + c * 32, o);
          tmem_ld_wait();
#pragma unroll
          for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * alpha);
          tmem_st32(tO + c * 32, o);
        }
      }
      // p = 2^(s * scale - m_used) as bf16 pairs over the first 32 of this
      // half's columns (chunk c's 32 scores are read before P of chunk c
      // covers columns 16 c .. 16 c + 15, whose scores are already used);
      // row sum in fp32
      const float2 scale2 = make_float2(p.scale_log2, p.scale_log2);
      const float2 negm2 = make_float2(-m_used, -m_used);
      float2 sm[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        uint32_t u[32], pk[16];
        tmem_ld32(tSh + 32 * c, u);
        tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const int k0 = 32 * c + 2 * i;
          const float2 x = __ffma2_rn(make_float2(__uint_as_float(u[2 * i]), __uint_as_float(u[2 * i + 1])),
                                      scale2, negm2);
          float2 e = make_float2(ex2_approx(x.x), ex2_approx(x.y));
          if (diag) {
            e.x = (k0 <= lim) ? e.x : 0.f;
            e.y = (k0 + 1 <= lim) ? e.y : 0.f;
          }
          sm[i & 1] = __fadd2_rn(sm[i & 1], e);
          pk[i] = pack_bf16x2(e.x, e.y);
        }
        tmem_st16(tSh + 16 * c, pk);
      }
      tmem_st_wait();
      l += (sm[0].x + sm[1].x) + (sm[0].y + sm[1].y);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(p_full0 + 8 * t);
    }
    // epilogue: O_t / l (both halves' sums) once the tile's last P V is done
    {
      const float l_all = l + exchange(l);
      if (ok) {
        int w = 0;
        if (lane == 0)
          w = mbar_wait_bounded(o_done0 + 8 * t, (pvc + qbt) & 1, abort_flag, p.err, p.timeout_ns);
        ok = __shfl_sync(0xffffffffu, w, 0) != 0;
      }
      pvc += qbt + 1;
      if (ok) {
        tc_fence_after();
        const float inv = 1.f / l_all;
        bf16* dst = p.out + (int64_t)(I.row0 + qi) * p.ld_out + (int64_t)I.h * HD + half * (HD / 2);
#pragma unroll 1
        for (int c = 0; c < HD / 64; ++c) {
          uint32_t o[32];
          tmem_ld32(tO + c * 32, o);
          tmem_ld_wait();
          if (qi < p.K) {
            float v[32];
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(o[i]) * inv;
#pragma unroll
            for (int i = 0; i < 4; ++i) store_vec(dst + c * 32 + 8 * i, v + 8 * i);
          }
        }
      }
      // O_t is read out: the next item's first P V may overwrite it
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(o_free0 + 8 * t);
    }
    }   // items
  }

  // Reconverge each warp first: in the producer and MMA warps only lane 0
  // ran the role loop, and the block barrier counts whole warps.
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, 512);
  }
}

// V^T of every key-value head: vt[((b * Hkv + g) * hd + e) * pad + j] =
// qkv[(b * K + j) * ld + col0 + g * hd + e]; the pad - K columns past the last
// key get zeros where a 16-byte store reaches them. Used when V^T is not
// produced by the QKV projection itself. Blocks stride over 64 x 64 tiles:
// 16-byte loads along e (eight threads per 128-byte row piece) into shared
// memory, then 16-byte stores along j. Needs hd, ld and col0 multiples of 8
// and 16-byte aligned pointers (checked by the caller).
constexpr int kVtTile = 64;
constexpr int kVtThreads = 256;
constexpr int kVtLd = kVtTile / 2 + 1;   // 32-bit words per shared row: odd, so column reads spread over banks

__global__ void __launch_bounds__(kVtThreads)
    vt_transpose_kernel(const bf16* qkv, int64_t ld, int col0, int B, int K, int Hkv, int hd,
                        int pad, bf16* vt) {
  __shared__ uint32_t tile[kVtTile * kVtLd];   // [j][e], two bf16 per word
  pdl_trigger();
  pdl_wait();
  const uint16_t* tile16 = reinterpret_cast<const uint16_t*>(tile);
  const int ntj = (K + kVtTile - 1) / kVtTile, nte = (hd + kVtTile - 1) / kVtTile;
  const int64_t ntiles = (int64_t)ntj * nte * B * Hkv;
  for (int64_t t = blockIdx.x; t < ntiles; t += gridDim.x) {
    const int j0 = (int)(t % ntj) * kVtTile;
    const int64_t r = t / ntj;
    const int e0 = (int)(r % nte) * kVtTile;
    const int64_t bg = r / nte;                     // b * Hkv + g
    const int g = (int)(bg % Hkv);
    const int64_t b = bg / Hkv;
    for (int c = threadIdx.x; c < kVtTile * 8; c += kVtThreads) {
      const int jj = c >> 3, ec = (c & 7) * 8;
      const int j = j0 + jj, e = e0 + ec;
      if (j < K && e + 8 <= hd) {
        const uint4 v = *reinterpret_cast<const uint4*>(qkv + (b * K + j) * ld + col0 + g * hd + e);
        uint32_t* w = tile + jj * kVtLd + ec / 2;
        w[0] = v.x;
        w[1] = v.y;
        w[2] = v.z;
        w[3] = v.w;
      }
    }
    __syncthreads();
    for (int c = threadIdx.x; c < kVtTile * 8; c += kVtThreads) {
      const int ee = c >> 3, jc = (c & 7) * 8;
      const int e = e0 + ee, j = j0 + jc;
      if (e < hd && j < K) {
        uint32_t o[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int ja = jc + 2 * i;
          const uint32_t lo = j0 + ja < K ? tile16[ja * 2 * kVtLd + ee] : 0u;
          const uint32_t hi = j0 + ja + 1 < K ? tile16[(ja + 1) * 2 * kVtLd + ee] : 0u;
          o[i] = lo | (hi << 16);
        }
        *reinterpret_cast<uint4*>(vt + (bg * hd + e) * pad + j) = make_uint4(o[0], o[1], o[2], o[3]);
      }
    }
    __syncthreads();
  }
}

template <int HD>
cudaError_t launch_attn(const void* qkv, int64_t ld_qkv, const void* vt, int pad, void* out,
                        int64_t ld_out, int B, int K, int Hq, int Hkv, const Dev& dev) {
  using C = AttnCfg<HD>;
  static int attr_done[64] = {0};
  int device = 0;
  cudaGetDevice(&device);
  if (device < 64 && !attr_done[device]) {
    cudaError_t e = cudaFuncSetAttribute(attn_tc_kernel<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         C::SMEM);
    if (e != cudaSuccess) return e;
    attr_done[device] = 1;
  }
  CUtensorMap tq, tv;
  if (!make_tmap_bf16(&tq, qkv, (uint64_t)B * K, (uint64_t)ld_qkv, (uint64_t)ld_qkv, 64, kQB) ||
      !make_tmap_bf16(&tv, vt, (uint64_t)B * Hkv * HD, (uint64_t)K, (uint64_t)pad, 64, HD))
    return cudaErrorInvalidValue;
  AttnDev p;
  p.K = K;
  p.B = B;
  p.Hq = Hq;
  p.Hkv = Hkv;
  p.q_dim = Hq * HD;
  p.scale_log2 = 1.4426950408889634f / sqrtf((float)HD);
  p.out = static_cast<bf16*>(out);
  p.ld_out = ld_out;
  p.err = dev.err;
  p.timeout_ns = kWaitTimeoutNs;
  const int nqb = (K + kQB - 1) / kQB;
  p.pair = (int64_t)((nqb + 1) / 2) * Hq * B >= dev.num_sms ? 1 : 0;
  // persistent: one CTA per SM (TMEM is allocated in full) over the work
  // items, each CTA taking every G-th item of the longest-first order
  const int64_t items = (int64_t)Hq * B * (p.pair ? (nqb + 1) / 2 : nqb);
  if (items > INT32_MAX) return cudaErrorInvalidValue;
  const int64_t grid = items < dev.num_sms ? items : dev.num_sms;
  return launch_pdl(attn_tc_kernel<HD>, dim3((unsigned)grid), dim3(kAttnThreads), C::SMEM, dev.stream, tq, tv, p);
}

}  // namespace

int vt_pad(int K) { return (K + 7) & ~7; }

cudaError_t vt_from_qkv(const void* qkv, int64_t ld_qkv, int col0, int B, int K, int Hkv, int hd,
                        void* vt, const Dev& dev) {
  if ((int64_t)B * Hkv * hd * K <= 0) return cudaSuccess;
  if (hd % 8 || ld_qkv % 8 || col0 % 8 || (reinterpret_cast<uintptr_t>(qkv) & 15) ||
      (reinterpret_cast<uintptr_t>(vt) & 15))
    return cudaErrorInvalidValue;
  const int64_t tiles = (int64_t)((K + kVtTile - 1) / kVtTile) * ((hd + kVtTile - 1) / kVtTile) * B * Hkv;
  const int64_t cap = 8 * (int64_t)dev.num_sms;   // 8 blocks of 256 threads per SM
  return launch_pdl(vt_transpose_kernel, dim3((unsigned)std::min(tiles, cap)), dim3(kVtThreads), 0,
                    dev.stream, static_cast<const bf16*>(qkv), ld_qkv, col0, B, K, Hkv,
                    hd, vt_pad(K), static_cast<bf16*>(vt));
}

cudaError_t attention_tc(const void* qkv, int64_t ld_qkv, const void* vt, void* out, int64_t ld_out,
                         int B, int K, int n_heads, int n_kv_heads, int head_dim, const Dev& dev) {
  if (B <= 0 || K <= 0) return cudaSuccess;
  if (head_dim == 64)
    return launch_attn<64>(qkv, ld_qkv, vt, vt_pad(K), out, ld_out, B, K, n_heads, n_kv_heads, dev);
  if (head_dim == 128)
    return launch_attn<128>(qkv, ld_qkv, vt, vt_pad(K), out, ld_out, B, K, n_heads, n_kv_heads, dev);
  return cudaErrorInvalidValue;
}

}  // namespace adadsf
