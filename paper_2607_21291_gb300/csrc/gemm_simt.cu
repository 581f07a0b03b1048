// fp32 projections on CUDA cores (FFMA), for fp32 storage. TF32 tensor-core
// rounding would not hold the fp32 tolerance, so fp32 models take this path.
// Same epilogue semantics as the tensor-core kernel (see internal.h).
#include "common.cuh"
#include "internal.h"

namespace adadsf {
namespace {

constexpr int TM = 64, TN = 64, TK = 16;

struct SimtDev {
  const float* A; int64_t lda;
  const float* W; const float* W2; int64_t ldw;
  int M, N, K;
  int act;
  const float* bias;
  const float* add_packed; int64_t ld_add_packed;
  const float* add_rows; int64_t ld_add_rows;
  const int32_t* rows;
  int out_mapped;
  float* out; int64_t ld_out;
  const float* gate;                        // score gate (see internal.h), or null
  const float* gbase; int64_t ld_gbase;
};

template <bool DUAL>
__global__ void __launch_bounds__(256) gemm_f32_kernel(const SimtDev p) {
  pdl_trigger();
  pdl_wait();
  __shared__ float As[TK][TM + 4];
  __shared__ float Ws[TK][TN + 4];
  __shared__ float W2s[DUAL ? TK : 1][TN + 4];
  const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
  const int row0 = blockIdx.y * TM, col0 = blockIdx.x * TN;
  float acc[4][4] = {}, acc2[4][4] = {};
  for (int k0 = 0; k0 < p.K; k0 += TK) {
    for (int i = threadIdx.x; i < TM * TK; i += 256) {
      const int r = i / TK, kk = i % TK;
      const int gm = row0 + r, gn = col0 + r, gk = k0 + kk;
      As[kk][r] = (gm < p.M && gk < p.K) ? p.A[(int64_t)gm * p.lda + gk] : 0.f;
      Ws[kk][r] = (gn < p.N && gk < p.K) ? p.W[(int64_t)gn * p.ldw + gk] : 0.f;
      if (DUAL) W2s[kk][r] = (gn < p.N && gk < p.K) ? p.W2[(int64_t)gn * p.ldw + gk] : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < TK; ++kk) {
      float a[4], b[4], b2[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        a[i] = As[kk][ty * 4 + i];
        b[i] = Ws[kk][tx * 4 + i];
        if (DUAL) b2[i] = W2s[kk][tx * 4 + i];
      }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
          if (DUAL) acc2[i][j] = fmaf(a[i], b2[j], acc2[i][j]);
        }
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int m = row0 + ty * 4 + i;
    if (m >= p.M) continue;
    const int64_t arow = p.rows ? (int64_t)p.rows[m] : (int64_t)m;
    if (arow < 0) continue;   // a row that bypasses the layer: nothing read or written
    const int64_t orow = p.out_mapped ? arow : (int64_t)m;
    const float g = p.gate ? 1.f / (1.f + expf(-p.gate[arow])) : 1.f;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = col0 + tx * 4 + j;
      if (n >= p.N) continue;
      float v = acc[i][j];
      if (p.bias) v += p.bias[n];
      if (DUAL) {
        v = v / (1.f + expf(-v)) * acc2[i][j];
      } else if (p.act == ACT_GELU) {
        v = 0.5f * v * (1.f + erff(v * 0.70710678118654752f));
      }
      if (p.add_packed) v += p.add_packed[(int64_t)m * p.ld_add_packed + n];
      if (p.gate && p.gbase) {
        const float b = p.gbase[arow * p.ld_gbase + n];
        v = fmaf(g, v - b, b);
      } else if (p.gate) {
        v = fmaf(g, v, p.add_rows[arow * p.ld_add_rows + n]);
      } else if (p.add_rows) {
        v += p.add_rows[arow * p.ld_add_rows + n];
      }
      p.out[orow * p.ld_out + n] = v;
    }
  }
}

}  // namespace

cudaError_t gemm_f32(const GemmArgs& a, const Dev& dev) {
  if (a.M <= 0) return cudaSuccess;
  if (a.K2 > 0 || a.epi.bias2 || a.a_gather || a.epi.nrm_psum) return cudaErrorInvalidValue;
  SimtDev p;
  p.A = static_cast<const float*>(a.A); p.lda = a.lda;
  p.W = static_cast<const float*>(a.W); p.W2 = static_cast<const float*>(a.W2); p.ldw = a.ldw;
  p.M = (int)a.M; p.N = a.N; p.K = a.K;
  p.act = a.epi.act;
  p.bias = static_cast<const float*>(a.epi.bias);
  p.add_packed = static_cast<const float*>(a.epi.add_packed); p.ld_add_packed = a.epi.ld_add_packed;
  p.add_rows = static_cast<const float*>(a.epi.add_rows); p.ld_add_rows = a.epi.ld_add_rows;
  p.rows = a.epi.rows;
  p.out_mapped = a.epi.out_mapped ? 1 : 0;
  p.out = static_cast<float*>(a.epi.out); p.ld_out = a.epi.ld_out;
  p.gate = a.epi.gate_scores;
  p.gbase = static_cast<const float*>(a.epi.gate_base); p.ld_gbase = a.epi.ld_gate_base;
  if (p.gate && (p.gbase ? p.add_rows != nullptr : p.add_rows == nullptr)) return cudaErrorInvalidValue;
  dim3 grid((a.N + TN - 1) / TN, (unsigned)((a.M + TM - 1) / TM));
  if (a.epi.act == ACT_SWIGLU)
    return launch_pdl(gemm_f32_kernel<true>, grid, dim3(256), 0, dev.stream, p);
  return launch_pdl(gemm_f32_kernel<false>, grid, dim3(256), 0, dev.stream, p);
}

}  // namespace adadsf
