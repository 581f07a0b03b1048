// Eq. 1 among the kept tokens on the 5th-generation tensor cores (bf16).
//
// One CTA per (128-query block, query head, sequence). Keys arrive in blocks
// of 128; attention is causal in packed order (kept positions ascend, so this
// is the original causal mask restricted to the kept set, Sec. 3.4).
//   warp 0     TMA: the Q tile once, then the K tile of each key block into a
//              2-stage ring released as soon as S of that block is done;
//   warp 10    TMA: the V^T tile of each key block into a 2-stage ring
//              released after P V (128-byte swizzled, K-major operands).
//   warp 1     allocates TMEM; one thread issues S = Q K^T into a double-
//              buffered TMEM S (tcgen05.mma, M = 128, N = 128) and, once the
//              softmax warps have written P, O += P V into TMEM O (N = hd).
//   warps 2-9  one query row and half of the key columns per thread (two
//              warps per TMEM lane quarter, exchanging row maxima and sums
//              through shared memory): read S from TMEM, mask, online
//              softmax in fp32 (exp2 with a row maximum held at most 2^8
//              below the true one, so O is rescaled only when the maximum
//              grows by more than that), write P as bf16 into one of two
//              swizzled operand tiles (so P of block j is written while
//              P V of block j-1 runs), and at the end O / l -> global.
// V enters as V^T (features x keys per key-value head), written by the QKV
// projection's epilogue, so both MMAs read K-major operands.
// Every barrier wait is bounded in time (device error word on give-up).
#include <cuda.h>

#include "common.cuh"
#include "internal.h"

namespace adadsf {
namespace {

constexpr int kQB = 128;            // queries per CTA = TMEM lanes
constexpr int kKB = 128;            // keys per block
constexpr int kSoftWarps = 8;       // two per TMEM lane quarter, each on 64 key columns
constexpr int kVWarp = 2 + kSoftWarps;   // warp loading the V^T tiles
constexpr int kAttnThreads = 32 * (kVWarp + 1);
constexpr float kRescaleLog2 = 8.f; // O rescaled only when the row max grows by > 2^8

template <int HD>
struct AttnCfg {
  static constexpr int HS = HD / 64;               // 64-feature slabs of a head row
  static constexpr int SLAB = kQB * 128;           // one 128-row x 128-byte slab
  static constexpr int Q_BYTES = HS * SLAB;
  static constexpr int K_BYTES = HS * SLAB;
  static constexpr int V_SLAB = HD * 128;          // HD feature rows x 64 keys
  static constexpr int V_BYTES = 2 * V_SLAB;       // 128 keys
  static constexpr int P_BYTES = 2 * SLAB;         // 128 queries x 128 keys
  static constexpr int DATA = Q_BYTES + 2 * K_BYTES + 2 * V_BYTES + 2 * P_BYTES;   // P double-buffered
  static constexpr int TAIL = 256 + 2048;         // barriers, then the softmax exchange area
  // Room left for aligning the dynamic base to 1024 bytes (the kernel checks
  // its actual misalignment); padded so that one CTA holds an SM (TMEM is
  // allocated in full).
  static constexpr int SLACK = (232448 - DATA - TAIL) < 1024 ? (232448 - DATA - TAIL) : 1024;
  static constexpr int SMEM_RAW = DATA + TAIL + SLACK;
  static constexpr int SMEM = SMEM_RAW > 120 * 1024 ? SMEM_RAW : 120 * 1024;
  static_assert(SLACK >= 256, "shared memory");
};

// 2^x on the SFU (ex2.approx.ftz.f32: relative error ~2^-22, flushes
// denormal results; P is rounded to bf16 afterwards).
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

struct AttnDev {
  int K;                 // kept tokens per sequence
  int Hq, Hkv, q_dim;
  float scale_log2;      // log2(e) / sqrt(hd)
  bf16* out;
  int64_t ld_out;
  int* err;
  unsigned long long timeout_ns;
};

template <int HD>
__global__ void __launch_bounds__(kAttnThreads, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tmQK, const __grid_constant__ CUtensorMap tmVt,
                   const AttnDev p) {
  using C = AttnCfg<HD>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  if (smem - smem_raw > C::SLACK) {   // the layout would not fit: report and touch nothing
    if (threadIdx.x == 0) set_device_error(p.err, DEVERR_TIMEOUT);
    return;
  }
  const uint32_t sQ = smem_u32(smem);
  const uint32_t sK0 = sQ + C::Q_BYTES;
  const uint32_t sV0 = sK0 + 2 * C::K_BYTES;
  const uint32_t sP0 = sV0 + 2 * C::V_BYTES;       // [2]
  uint8_t* sP_ptr = smem + (sP0 - sQ);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::DATA);
  const uint32_t b0 = smem_u32(bars);
  const uint32_t q_full = b0;
  const uint32_t k_full0 = b0 + 8;       // [2] K ring: free once S of the block is done
  const uint32_t k_empty0 = b0 + 24;     // [2]
  const uint32_t s_full0 = b0 + 40;      // [2]
  const uint32_t s_free0 = b0 + 56;      // [2]
  const uint32_t p_full0 = b0 + 72;      // [2] per P buffer
  const uint32_t pv_done0 = b0 + 88;     // [2] per P buffer
  const uint32_t drain = b0 + 104;
  const uint32_t pair0 = b0 + 112;       // [4] the two softmax warps of a lane quarter
  const uint32_t v_full0 = b0 + 144;     // [2] V^T ring: free once P V of the block is done
  const uint32_t v_empty0 = b0 + 160;    // [2]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 22);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  // per quarter, per exchange slot (2), per half: one float per lane
  float* xchg = reinterpret_cast<float*>(smem + C::DATA + 256);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int nqb = (p.K + kQB - 1) / kQB;
  const int qb = nqb - 1 - (int)blockIdx.x;   // longest rows first
  const int h = blockIdx.y, b = blockIdx.z;
  const int g = h / (p.Hq / p.Hkv);
  const int n_kv = qb + 1;
  const int row0 = b * p.K;

  pdl_trigger();
  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(k_full0 + 8 * i, 1);
      mbar_init(k_empty0 + 8 * i, 1);
      mbar_init(v_full0 + 8 * i, 1);
      mbar_init(v_empty0 + 8 * i, 1);
      mbar_init(s_full0 + 8 * i, 1);
      mbar_init(s_free0 + 8 * i, kSoftWarps);
      mbar_init(p_full0 + 8 * i, kSoftWarps);
      mbar_init(pv_done0 + 8 * i, 1);
    }
    for (int i = 0; i < 4; ++i) mbar_init(pair0 + 8 * i, 2);
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
  const uint32_t tS = tmem_base;          // S buffers at columns 0 and 128
  const uint32_t tO = tmem_base + 256;    // O at columns 256 .. 256 + HD

  if (warp == 0 || warp == kVWarp) {
    // ------------------------------------------------------------ TMA producers
    // warp 0: Q once, then the K ring; warp kVWarp: the V^T ring
    if (lane == 0) {
      const bool kprod = warp == 0;
      pdl_wait();
      if (kprod) {
        mbar_arrive_expect_tx(q_full, C::Q_BYTES);
        for (int s = 0; s < C::HS; ++s)
          tma_load_2d(sQ + s * C::SLAB, &tmQK, h * HD + s * 64, row0 + qb * kQB, q_full);
      }
      const uint32_t full0 = kprod ? k_full0 : v_full0;
      const uint32_t empty0 = kprod ? k_empty0 : v_empty0;
      int issued = 0;
      for (int j = 0; j < n_kv; ++j) {
        const int st = j & 1;
        if (!mbar_wait_bounded(empty0 + 8 * st, ((j >> 1) & 1) ^ 1, abort_flag, p.err, p.timeout_ns))
          break;
        const uint32_t fb = full0 + 8 * st;
        if (kprod) {
          mbar_arrive_expect_tx(fb, C::K_BYTES);
          for (int s = 0; s < C::HS; ++s)
            tma_load_2d(sK0 + st * C::K_BYTES + s * C::SLAB, &tmQK, p.q_dim + g * HD + s * 64,
                        row0 + j * kKB, fb);
        } else {
          mbar_arrive_expect_tx(fb, C::V_BYTES);
          for (int ks = 0; ks < 2; ++ks)
            tma_load_2d(sV0 + st * C::V_BYTES + ks * C::V_SLAB, &tmVt, j * kKB + ks * 64,
                        (b * p.Hkv + g) * HD, fb);
        }
        ++issued;
      }
      // drain: the copies issued last into each stage have landed
      if (kprod) mbar_wait_drain(q_full, 0, p.timeout_ns);
      for (int st = 0; st < 2 && st < issued; ++st) {
        const int last = st + ((issued - 1 - st) / 2) * 2;
        mbar_wait_drain(full0 + 8 * st, (uint32_t)((last >> 1) & 1), p.timeout_ns);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc_s = idesc_bf16_f32(kQB, kKB);
      constexpr uint32_t idesc_o = idesc_bf16_f32(kQB, HD);
      bool ok = mbar_wait_bounded(q_full, 0, abort_flag, p.err, p.timeout_ns);
      for (int j = 0; ok && j <= n_kv; ++j) {
        if (j < n_kv) {
          const int st = j & 1;
          if (!mbar_wait_bounded(k_full0 + 8 * st, (j >> 1) & 1, abort_flag, p.err, p.timeout_ns) ||
              (j >= 2 && !mbar_wait_bounded(s_free0 + 8 * st, ((j >> 1) - 1) & 1, abort_flag, p.err,
                                            p.timeout_ns))) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t kst = sK0 + st * C::K_BYTES;
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk) {
            const uint32_t off = (kk >> 2) * C::SLAB + (kk & 3) * 32;
            tc_mma_f16(tS + st * kKB, smem_desc_sw128(sQ + off), smem_desc_sw128(kst + off), idesc_s,
                       kk > 0 ? 1u : 0u);
          }
          tc_commit(s_full0 + 8 * st);
          tc_commit(k_empty0 + 8 * st);   // K tile consumed
        }
        if (j >= 1) {
          const int jj = j - 1, pb = jj & 1;   // V^T stage and P buffer of block jj
          if (!mbar_wait_bounded(p_full0 + 8 * pb, (jj >> 1) & 1, abort_flag, p.err, p.timeout_ns) ||
              !mbar_wait_bounded(v_full0 + 8 * pb, (jj >> 1) & 1, abort_flag, p.err, p.timeout_ns)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t vst = sV0 + pb * C::V_BYTES;
          const uint32_t pst = sP0 + pb * C::P_BYTES;
#pragma unroll
          for (int kk = 0; kk < kKB / 16; ++kk) {
            tc_mma_f16(tO, smem_desc_sw128(pst + (kk >> 2) * C::SLAB + (kk & 3) * 32),
                       smem_desc_sw128(vst + (kk >> 2) * C::V_SLAB + (kk & 3) * 32), idesc_o,
                       (jj > 0 || kk > 0) ? 1u : 0u);
          }
          tc_commit(pv_done0 + 8 * pb);
          tc_commit(v_empty0 + 8 * pb);
        }
      }
      tc_commit(drain);
      mbar_wait_drain(drain, 0, p.timeout_ns);
    }
  } else {
    // ------------------------------------------------------------ softmax (warps 2..9)
    pdl_wait();
    const int quarter = warp & 3;
    const int half = (warp - 2) >> 2;              // key columns [64 half, 64 half + 64)
    const int r = quarter * 32 + lane;             // query row in the block = TMEM lane
    const int qi = qb * kQB + r;                   // query index in the sequence
    const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;
    const uint32_t pairbar = pair0 + 8 * quarter;
    uint32_t xk = 0;                               // exchanges done with the partner warp
    // value of the partner warp (same rows, other half) for this exchange
    auto exchange = [&](float mine, float* theirs) -> bool {
      float* slot = xchg + ((quarter * 2 + (xk & 1)) * 2) * 32;
      slot[half * 32 + lane] = mine;
      __syncwarp();
      int w = 1;
      if (lane == 0) {
        mbar_arrive(pairbar);
        w = mbar_wait_bounded(pairbar, xk & 1, abort_flag, p.err, p.timeout_ns);
      }
      ++xk;
      if (!__shfl_sync(0xffffffffu, w, 0)) return false;
      *theirs = slot[(half ^ 1) * 32 + lane];
      return true;
    };
    float m_used = -INFINITY, l = 0.f;
    bool ok = true;
    for (int j = 0; j < n_kv && ok; ++j) {
      const int st = j & 1;
      int w = 0;
      if (lane == 0) w = mbar_wait_bounded(s_full0 + 8 * st, (j >> 1) & 1, abort_flag, p.err, p.timeout_ns);
      if (!__shfl_sync(0xffffffffu, w, 0)) { ok = false; break; }
      tc_fence_after();
      const uint32_t s_row = tS + lane_off + st * kKB + half * 64;
      // keys above lim (relative to this half) are masked: diagonal block only
      const int lim = (j == qb) ? qi - j * kKB - half * 64 : kKB;
      // pass 1: row maximum of the raw scores (scale > 0) over both halves
      float mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll 1
      for (int c = 0; c < 2; ++c) {
        uint32_t u[32];
        tmem_ld32(s_row + c * 32, u);
        tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const float v = (c * 32 + i <= lim) ? __uint_as_float(u[i]) : -INFINITY;
          mx[i & 3] = fmaxf(mx[i & 3], v);
        }
      }
      float part = fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])), other;
      if (!exchange(part, &other)) { ok = false; break; }
      const float bmax = fmaxf(part, other) * p.scale_log2;
      bool need = false;
      if (j == 0) m_used = bmax;
      else need = bmax > m_used + kRescaleLog2;
      const int pb = j & 1;
      // P buffer pb is free once P V of block j - 2 has completed
      if (j >= 2) {
        int w2 = 0;
        if (lane == 0)
          w2 = mbar_wait_bounded(pv_done0 + 8 * pb, ((j >> 1) - 1) & 1, abort_flag, p.err, p.timeout_ns);
        if (!__shfl_sync(0xffffffffu, w2, 0)) { ok = false; break; }
      }
      if (__any_sync(0xffffffffu, need)) {
        // O is stable once P V of block j - 1 has completed; each half
        // rescales its half of the O columns
        int w3 = 0;
        if (lane == 0)
          w3 = mbar_wait_bounded(pv_done0 + 8 * (pb ^ 1), ((j - 1) >> 1) & 1, abort_flag, p.err,
                                 p.timeout_ns);
        if (!__shfl_sync(0xffffffffu, w3, 0)) { ok = false; break; }
        const float alpha = need ? ex2_approx(m_used - bmax) : 1.f;
        if (need) {
          l *= alpha;
          m_used = bmax;
        }
        tc_fence_after();
#pragma unroll 1
        for (int c = 0; c < HD / 64; ++c) {
          const uint32_t ta = tO + lane_off + half * (HD / 2) + c * 32;
          uint32_t u[32];
          tmem_ld32(ta, u);
          tmem_ld_wait();
#pragma unroll
          for (int i = 0; i < 32; ++i) u[i] = __float_as_uint(__uint_as_float(u[i]) * alpha);
          tmem_st32(ta, u);
        }
        tmem_st_wait();
      }
      // pass 2: p = 2^(s * scale - m_used), partial row sum, this half's 64
      // keys of P row r as bf16 into slab `half` (16-byte chunks XOR-swizzled)
      uint8_t* prow = sP_ptr + pb * C::P_BYTES + half * C::SLAB + r * 128;
      float sm[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 1
      for (int c = 0; c < 2; ++c) {
        uint32_t u[32];
        tmem_ld32(s_row + c * 32, u);
        tmem_ld_wait();
        float e[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const float t = ex2_approx(fmaf(__uint_as_float(u[i]), p.scale_log2, -m_used));
          e[i] = (c * 32 + i <= lim) ? t : 0.f;
          sm[i & 3] += e[i];
        }
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const int ch = c * 4 + k;
          const float* q = e + 8 * k;
          *reinterpret_cast<uint4*>(prow + ((ch ^ (r & 7)) << 4)) =
              make_uint4(pack_bf16x2(q[0], q[1]), pack_bf16x2(q[2], q[3]), pack_bf16x2(q[4], q[5]),
                         pack_bf16x2(q[6], q[7]));
        }
      }
      l += (sm[0] + sm[1]) + (sm[2] + sm[3]);
      fence_proxy_async_smem();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(s_free0 + 8 * st);   // S buffer may be overwritten
        mbar_arrive(p_full0 + 8 * pb);
      }
    }
    // epilogue: O / (l of both halves); each half stores its HD/2 columns
    float l_other = 0.f;
    if (ok) ok = exchange(l, &l_other);
    if (ok) {
      int w = 0;
      if (lane == 0)
        w = mbar_wait_bounded(pv_done0 + 8 * ((n_kv - 1) & 1), ((n_kv - 1) >> 1) & 1, abort_flag, p.err,
                              p.timeout_ns);
      ok = __shfl_sync(0xffffffffu, w, 0) != 0;
    }
    if (ok) {
      tc_fence_after();
      const float inv = 1.f / (l + l_other);
      bf16* dst = p.out + (int64_t)(row0 + qi) * p.ld_out + (int64_t)h * HD + half * (HD / 2);
#pragma unroll 1
      for (int c = 0; c < HD / 64; ++c) {
        uint32_t u[32];
        tmem_ld32(tO + lane_off + half * (HD / 2) + c * 32, u);
        tmem_ld_wait();
        if (qi < p.K) {
          float v[32];
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(u[i]) * inv;
#pragma unroll
          for (int i = 0; i < 4; ++i) store_vec(dst + c * 32 + 8 * i, v + 8 * i);
        }
      }
    }
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
// qkv[(b * K + j) * ld + col0 + g * hd + e]. Used when V^T is not produced by
// the QKV projection itself.
__global__ void vt_transpose_kernel(const bf16* qkv, int64_t ld, int col0, int B, int K, int Hkv,
                                    int hd, int pad, bf16* vt) {
  pdl_trigger();
  pdl_wait();
  const int64_t n = (int64_t)B * Hkv * hd * K;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int j = (int)(i % K);
    const int64_t re = i / K;                       // (b * Hkv + g) * hd + e
    const int e = (int)(re % hd);
    const int64_t bg = re / hd;
    const int g = (int)(bg % Hkv), b = (int)(bg / Hkv);
    vt[re * pad + j] = qkv[((int64_t)b * K + j) * ld + col0 + g * hd + e];
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
  p.Hq = Hq;
  p.Hkv = Hkv;
  p.q_dim = Hq * HD;
  p.scale_log2 = 1.4426950408889634f / sqrtf((float)HD);
  p.out = static_cast<bf16*>(out);
  p.ld_out = ld_out;
  p.err = dev.err;
  p.timeout_ns = kWaitTimeoutNs;
  dim3 grid((K + kQB - 1) / kQB, Hq, B);
  return launch_pdl(attn_tc_kernel<HD>, grid, dim3(kAttnThreads), C::SMEM, dev.stream, tq, tv, p);
}

}  // namespace

int vt_pad(int K) { return (K + 7) & ~7; }

cudaError_t vt_from_qkv(const void* qkv, int64_t ld_qkv, int col0, int B, int K, int Hkv, int hd,
                        void* vt, const Dev& dev) {
  const int64_t n = (int64_t)B * Hkv * hd * K;
  if (n <= 0) return cudaSuccess;
  const int64_t blocks = (n + 255) / 256;
  return launch_pdl(vt_transpose_kernel, dim3((unsigned)(blocks < 65535 * 8 ? blocks : 65535 * 8)),
                    dim3(256), 0, dev.stream, static_cast<const bf16*>(qkv), ld_qkv, col0, B, K, Hkv,
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
