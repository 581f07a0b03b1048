// Eq. 1 among the kept tokens of each sequence: softmax(Q K^T / sqrt(d_k)) V,
// causal in packed order. Kept positions ascend, so packed order is original
// order and "key j <= query i" is the original causal mask restricted to the
// kept set (Sec. 3.4: unselected tokens contribute no keys or values).
//
// bf16: flash-attention style, one CTA per (64-query block, head, sequence),
// 4 warps x 16 query rows, 64-key tiles double-buffered through shared memory
// with cp.async, S and O on warp-level bf16 MMAs with fp32 accumulation and an
// online softmax in fp32.
// fp32: one warp per (query, head), exact fp32 online softmax.
#include "common.cuh"
#include "internal.h"

namespace adadsf {
namespace {

constexpr int BQ = 64, BKV = 64;

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, int src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src),
               "r"(src_bytes)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                          uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
// c += a (16x16 bf16, row) * b (16x8 bf16, col), fp32 accumulate.
__device__ __forceinline__ void mma_bf16(float* c, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Element offset of 16-byte chunk c of row r in a swizzled [rows][HD] tile.
template <int HD>
__device__ __forceinline__ int swz(int r, int c) {
  return r * HD + ((c ^ (r & 7)) << 3);
}

// Rows [r0, r0 + 64) of a [K, HD] slice (row stride ld elements) into a
// swizzled tile; rows at or beyond K are zero-filled.
template <int HD>
__device__ __forceinline__ void load_tile(bf16* tile, const bf16* src, int64_t ld, int r0, int K) {
  constexpr int CH = HD / 8;
  for (int i = threadIdx.x; i < 64 * CH; i += 128) {
    const int r = i / CH, c = i % CH;
    const int gr = r0 + r;
    const bool ok = gr < K;
    const bf16* p = src + (int64_t)(ok ? gr : 0) * ld + c * 8;
    cp_async16(smem_u32(tile + swz<HD>(r, c)), p, ok ? 16 : 0);
  }
}

template <int HD>
__global__ void __launch_bounds__(128) attn_bf16_kernel(const bf16* qkv, int64_t ldq, bf16* out,
                                                        int64_t ldo, int K, int n_heads, int n_kv,
                                                        float scale_log2) {
  pdl_trigger();
  extern __shared__ __align__(128) uint8_t smem_raw[];
  bf16* sQ = reinterpret_cast<bf16*>(smem_raw);
  bf16* sK = sQ + BQ * HD;               // [2][BKV][HD]
  bf16* sV = sK + 2 * BKV * HD;          // [2][BKV][HD]

  const int nqb = (K + BQ - 1) / BQ;
  const int qb = nqb - 1 - (int)blockIdx.x;   // longest rows first
  const int h = blockIdx.y, b = blockIdx.z;
  const int g = h / (n_heads / n_kv);
  const int64_t row0 = (int64_t)b * K;
  const bf16* Qg = qkv + row0 * ldq + (int64_t)h * HD;
  const bf16* Kg = qkv + row0 * ldq + (int64_t)n_heads * HD + (int64_t)g * HD;
  const bf16* Vg = qkv + row0 * ldq + (int64_t)(n_heads + n_kv) * HD + (int64_t)g * HD;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  pdl_wait();
  load_tile<HD>(sQ, Qg, ldq, qb * BQ, K);
  load_tile<HD>(sK, Kg, ldq, 0, K);
  load_tile<HD>(sV, Vg, ldq, 0, K);
  cp_async_commit();

  float o[HD / 8][4];
#pragma unroll
  for (int i = 0; i < HD / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float m_i[2] = {-INFINITY, -INFINITY}, l_i[2] = {0.f, 0.f};
  uint32_t qf[HD / 16][4];

  const int n_blocks = qb + 1;
  for (int j = 0; j < n_blocks; ++j) {
    const int st = j & 1;
    if (j + 1 < n_blocks) {
      load_tile<HD>(sK + (st ^ 1) * BKV * HD, Kg, ldq, (j + 1) * BKV, K);
      load_tile<HD>(sV + (st ^ 1) * BKV * HD, Vg, ldq, (j + 1) * BKV, K);
    }
    cp_async_commit();
    cp_async_wait<1>();
    __syncthreads();
    if (j == 0) {
#pragma unroll
      for (int kk = 0; kk < HD / 16; ++kk) {
        const int r = warp * 16 + (lane & 7) + (((lane >> 3) & 1) << 3);
        const int c = kk * 2 + (lane >> 4);
        ldsm_x4(smem_u32(sQ + swz<HD>(r, c)), qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3]);
      }
    }
    const bf16* tK = sK + st * BKV * HD;
    const bf16* tV = sV + st * BKV * HD;

    // S = Q K^T for this warp's 16 rows x 64 keys
    float s[8][4];
#pragma unroll
    for (int i = 0; i < 8; ++i) s[i][0] = s[i][1] = s[i][2] = s[i][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) {
#pragma unroll
      for (int nb2 = 0; nb2 < 4; ++nb2) {
        const int r = nb2 * 16 + (lane & 7) + ((lane >> 4) << 3);
        const int c = kk * 2 + ((lane >> 3) & 1);
        uint32_t b0, b1, b2, b3;
        ldsm_x4(smem_u32(tK + swz<HD>(r, c)), b0, b1, b2, b3);
        mma_bf16(s[2 * nb2], qf[kk], b0, b1);
        mma_bf16(s[2 * nb2 + 1], qf[kk], b2, b3);
      }
    }
    // causal mask on the diagonal block
    if (j == qb) {
      const int q0 = qb * BQ + warp * 16 + (lane >> 2);
#pragma unroll
      for (int nb = 0; nb < 8; ++nb) {
        const int k0 = j * BKV + nb * 8 + 2 * (lane & 3);
        if (k0 > q0) s[nb][0] = -INFINITY;
        if (k0 + 1 > q0) s[nb][1] = -INFINITY;
        if (k0 > q0 + 8) s[nb][2] = -INFINITY;
        if (k0 + 1 > q0 + 8) s[nb][3] = -INFINITY;
      }
    }
    // online softmax (rows lane/4 and lane/4 + 8)
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      float mx = -INFINITY;
#pragma unroll
      for (int nb = 0; nb < 8; ++nb) mx = fmaxf(mx, fmaxf(s[nb][2 * r], s[nb][2 * r + 1]));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
      const float m_new = fmaxf(m_i[r], mx);
      const float ms = m_new == -INFINITY ? 0.f : m_new * scale_log2;
      const float alpha = exp2f(m_i[r] * scale_log2 - ms);
      m_i[r] = m_new;
      l_i[r] *= alpha;
#pragma unroll
      for (int i = 0; i < HD / 8; ++i) {
        o[i][2 * r] *= alpha;
        o[i][2 * r + 1] *= alpha;
      }
      float rs = 0.f;
#pragma unroll
      for (int nb = 0; nb < 8; ++nb) {
        s[nb][2 * r] = exp2f(s[nb][2 * r] * scale_log2 - ms);
        s[nb][2 * r + 1] = exp2f(s[nb][2 * r + 1] * scale_log2 - ms);
        rs += s[nb][2 * r] + s[nb][2 * r + 1];
      }
      l_i[r] += rs;
    }
    // O += P V
#pragma unroll
    for (int kk2 = 0; kk2 < 4; ++kk2) {
      uint32_t a[4];
      a[0] = pack_bf16x2(s[2 * kk2][0], s[2 * kk2][1]);
      a[1] = pack_bf16x2(s[2 * kk2][2], s[2 * kk2][3]);
      a[2] = pack_bf16x2(s[2 * kk2 + 1][0], s[2 * kk2 + 1][1]);
      a[3] = pack_bf16x2(s[2 * kk2 + 1][2], s[2 * kk2 + 1][3]);
#pragma unroll
      for (int nd2 = 0; nd2 < HD / 16; ++nd2) {
        const int r = kk2 * 16 + (lane & 7) + (((lane >> 3) & 1) << 3);
        const int c = nd2 * 2 + (lane >> 4);
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(smem_u32(tV + swz<HD>(r, c)), b0, b1, b2, b3);
        mma_bf16(o[2 * nd2], a, b0, b1);
        mma_bf16(o[2 * nd2 + 1], a, b2, b3);
      }
    }
    __syncthreads();
  }

  // finalize
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    float l = l_i[r];
    l += __shfl_xor_sync(0xffffffffu, l, 1);
    l += __shfl_xor_sync(0xffffffffu, l, 2);
    const float inv = 1.f / l;
    const int q = qb * BQ + warp * 16 + (lane >> 2) + 8 * r;
    if (q < K) {
      bf16* dst = out + (row0 + q) * ldo + (int64_t)h * HD + 2 * (lane & 3);
#pragma unroll
      for (int nd = 0; nd < HD / 8; ++nd) {
        *reinterpret_cast<uint32_t*>(dst + nd * 8) =
            pack_bf16x2(o[nd][2 * r] * inv, o[nd][2 * r + 1] * inv);
      }
    }
  }
}

// fp32: one warp per (query, head, sequence); lanes split the head dimension.
template <int HD>
__global__ void __launch_bounds__(128) attn_f32_kernel(const float* qkv, int64_t ldq, float* out,
                                                       int64_t ldo, int K, int n_heads, int n_kv,
                                                       float scale) {
  pdl_trigger();
  pdl_wait();
  constexpr int PL = HD / 32;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int i = blockIdx.x * 4 + warp;
  const int h = blockIdx.y, b = blockIdx.z;
  if (i >= K) return;
  const int g = h / (n_heads / n_kv);
  const int64_t row0 = (int64_t)b * K;
  const float* q = qkv + (row0 + i) * ldq + (int64_t)h * HD;
  float qv[PL], o[PL];
#pragma unroll
  for (int e = 0; e < PL; ++e) {
    qv[e] = q[lane + 32 * e];
    o[e] = 0.f;
  }
  float m = -INFINITY, l = 0.f;
  for (int jj = 0; jj <= i; ++jj) {
    const float* kr = qkv + (row0 + jj) * ldq + (int64_t)n_heads * HD + (int64_t)g * HD;
    const float* vr = qkv + (row0 + jj) * ldq + (int64_t)(n_heads + n_kv) * HD + (int64_t)g * HD;
    float d = 0.f;
#pragma unroll
    for (int e = 0; e < PL; ++e) d = fmaf(qv[e], kr[lane + 32 * e], d);
    const float sc = warp_sum(d) * scale;
    const float m_new = fmaxf(m, sc);
    const float a = expf(m - m_new);
    const float p = expf(sc - m_new);
    l = l * a + p;
#pragma unroll
    for (int e = 0; e < PL; ++e) o[e] = o[e] * a + p * vr[lane + 32 * e];
    m = m_new;
  }
  float* dst = out + (row0 + i) * ldo + (int64_t)h * HD;
#pragma unroll
  for (int e = 0; e < PL; ++e) dst[lane + 32 * e] = o[e] / l;
}

template <int HD>
cudaError_t launch_bf16(const bf16* qkv, int64_t ldq, bf16* out, int64_t ldo, int B, int K, int H,
                        int Hkv, const Dev& dev) {
  const size_t smem = (size_t)(BQ + 4 * BKV) * HD * sizeof(bf16);
  static int attr_done[64] = {0};
  int device = 0;
  cudaGetDevice(&device);
  if (device < 64 && !attr_done[device]) {
    cudaError_t e = cudaFuncSetAttribute(attn_bf16_kernel<HD>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    attr_done[device] = 1;
  }
  dim3 grid((K + BQ - 1) / BQ, H, B);
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)HD);
  return launch_pdl(attn_bf16_kernel<HD>, grid, dim3(128), smem, dev.stream, qkv, ldq, out, ldo, K,
                    H, Hkv, scale_log2);
}

}  // namespace

cudaError_t attention(int dtype, const void* qkv, int64_t ld_qkv, void* out, int64_t ld_out, int B,
                      int K, int n_heads, int n_kv_heads, int head_dim, const Dev& dev) {
  if (B <= 0 || K <= 0) return cudaSuccess;
  if (dtype == kBF16) {
    const bf16* q = static_cast<const bf16*>(qkv);
    bf16* o = static_cast<bf16*>(out);
    if (head_dim == 64) return launch_bf16<64>(q, ld_qkv, o, ld_out, B, K, n_heads, n_kv_heads, dev);
    if (head_dim == 128) return launch_bf16<128>(q, ld_qkv, o, ld_out, B, K, n_heads, n_kv_heads, dev);
    return cudaErrorInvalidValue;
  }
  const float* q = static_cast<const float*>(qkv);
  float* o = static_cast<float*>(out);
  dim3 grid((K + 3) / 4, n_heads, B);
  const float scale = 1.f / sqrtf((float)head_dim);
  if (head_dim == 64)
    return launch_pdl(attn_f32_kernel<64>, grid, dim3(128), 0, dev.stream, q, ld_qkv, o, ld_out, K,
                      n_heads, n_kv_heads, scale);
  if (head_dim == 128)
    return launch_pdl(attn_f32_kernel<128>, grid, dim3(128), 0, dev.stream, q, ld_qkv, o, ld_out, K,
                      n_heads, n_kv_heads, scale);
  return cudaErrorInvalidValue;
}

}  // namespace adadsf
