// Per-sequence Top-K of router scores (Sec. 3.4) as block-level device code:
// a radix select of the K-th largest score and the in-order emission of the
// kept positions. Shared by the stand-alone Top-K kernels and the fused
// router + Top-K kernel. Every function runs on a group of NT threads (whole
// warps, thread ids tid = 0..NT-1) that synchronise through `sync()`: the
// whole block (__syncthreads) or a named barrier of a subset of its warps.
#pragma once

#include <stdint.h>

namespace adadsf {

// Order-preserving key of an fp32 score: larger score -> larger key; -0.0 is
// folded onto +0.0; NaN maps to 0, below every number (-inf maps to 0x007FFFFF).
__device__ __forceinline__ uint32_t score_key(float f) {
  if (f != f) return 0u;
  uint32_t u = __float_as_uint(f);
  if ((u << 1) == 0u) u = 0u;   // -0.0 -> +0.0
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Exclusive prefix sum over the group of one int per thread; also returns
// the group total. warp_tot: NT / 32 + 1 ints of shared memory.
template <int NT, typename Sync>
__device__ __forceinline__ int group_excl_scan(int v, int* warp_tot, int& total, int tid, Sync sync) {
  constexpr int NW = NT / 32;
  static_assert(NT % 32 == 0 && NW <= 32, "group size");
  const int lane = tid & 31, w = tid >> 5;
  int incl = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int t = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += t;
  }
  if (lane == 31) warp_tot[w] = incl;
  sync();
  if (w == 0) {
    int t = lane < NW ? warp_tot[lane] : 0;
    int ti = t;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int u = __shfl_up_sync(0xffffffffu, ti, o);
      if (lane >= o) ti += u;
    }
    if (lane < NW) warp_tot[lane] = ti - t;   // exclusive prefix of warp totals
    if (lane == 31) warp_tot[NW] = ti;
  }
  sync();
  const int res = warp_tot[w] + incl - v;
  total = warp_tot[NW];
  sync();
  return res;
}

// Shared state of the group-wide Top-K.
struct TopkShared {
  int hist[2][256];     // alternate passes use alternate histograms
  int warp_tot[33];
  uint32_t digit[4];    // per pass, so no pass overwrites what another still reads
  int remaining[4];
};

// Radix select over the T order-preserving keys in shared memory (4 passes
// of 8 bits, most significant first): the K-th largest key `kth` and how many
// keys equal to it are kept (need_eq, lowest positions first). K >= 1. Two
// group barriers per pass: the next pass's histogram is cleared while this
// pass's is filled.
template <int NT, typename Sync>
__device__ __forceinline__ void radix_select(const uint32_t* keys, int T, int K, TopkShared& sh,
                                             uint32_t& kth, int& need_eq, int tid, Sync sync) {
  uint32_t prefix = 0, pmask = 0;
  int remaining = K;   // keys still to take at or below the current prefix
  for (int i = tid; i < 256; i += NT) sh.hist[0][i] = 0;
  sync();
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = 24 - 8 * pass;
    int* hist = sh.hist[pass & 1];
    for (int i = tid; i < 256; i += NT) sh.hist[(pass + 1) & 1][i] = 0;
    // Scores of one sequence tend to share their leading bits, so many keys
    // hit the same bin: the lanes of a warp with equal digits add once.
    for (int t0 = 0; t0 < T; t0 += NT) {
      const int t = t0 + tid;
      const uint32_t k = t < T ? keys[t] : 0u;
      const bool in = t < T && (k & pmask) == prefix;
      const uint32_t dg = (k >> shift) & 255u;
      const uint32_t peers = __match_any_sync(0xffffffffu, in ? dg : 0x100u);
      if (in && (tid & 31) == __ffs(peers) - 1) atomicAdd(&hist[dg], __popc(peers));
    }
    sync();
    if (tid < 32) {
      // lane l owns digits 255-8l .. 248-8l (descending)
      const int lane = tid;
      int cnt[8], lsum = 0;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        cnt[j] = hist[255 - 8 * lane - j];
        lsum += cnt[j];
      }
      int incl = lsum;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int t = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += t;
      }
      const int excl = incl - lsum;   // keys with a larger digit than this lane's
      const bool here = excl < remaining && incl >= remaining;
      if (here) {
        int above = excl;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          if (above + cnt[j] >= remaining) {
            sh.digit[pass] = (uint32_t)(255 - 8 * lane - j);
            sh.remaining[pass] = remaining - above;
            break;
          }
          above += cnt[j];
        }
      }
    }
    sync();
    prefix |= sh.digit[pass] << shift;
    pmask |= 255u << shift;
    remaining = sh.remaining[pass];
  }
  kth = prefix;
  need_eq = remaining;
}

// Calls emit(i, t) for the kept positions t in ascending order, i = 0..K-1:
// keys above kth, and the first need_eq keys equal to it. Each thread owns a
// contiguous chunk of positions; one group scan of the packed counts
// (above << 16 | equal; T <= 16384) places every chunk's output.
template <int NT, typename Sync, typename Emit>
__device__ __forceinline__ void emit_kept(const uint32_t* keys, int T, uint32_t kth, int need_eq,
                                          TopkShared& sh, int tid, Sync sync, Emit emit) {
  const int chunk = (T + NT - 1) / NT;
  const int t0 = min(T, tid * chunk), t1 = min(T, t0 + chunk);
  int n_gt = 0, n_eq = 0;
  for (int t = t0; t < t1; ++t) {
    n_gt += keys[t] > kth;
    n_eq += keys[t] == kth;
  }
  int total;
  const int base = group_excl_scan<NT>((n_gt << 16) | n_eq, sh.warp_tot, total, tid, sync);
  const int eq_base = base & 0xffff;   // equal keys before my chunk
  int out = (base >> 16) + min(eq_base, need_eq);
  int er = eq_base;
  for (int t = t0; t < t1; ++t) {
    const uint32_t k = keys[t];
    bool take = k > kth;
    if (k == kth) {
      take = er < need_eq;
      ++er;
    }
    if (take) emit(out++, t);
  }
}

constexpr int kMaxTopkT = 16384;   // sequence length limit of the Top-K code (packed counts)

}  // namespace adadsf
