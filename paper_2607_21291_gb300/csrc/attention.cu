// Eq. 1 among the kept tokens of each sequence, fp32 storage: softmax(Q K^T /
// sqrt(d_k)) V, causal in packed order. Kept positions ascend, so packed order
// is original order and "key j <= query i" is the original causal mask
// restricted to the kept set (Sec. 3.4: unselected tokens contribute no keys
// or values). One warp per (query, head), exact fp32 online softmax.
// (bf16 storage runs on the tensor cores: attention_tc.cu.)
#include "common.cuh"
#include "internal.h"

namespace adadsf {
namespace {

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

}  // namespace

cudaError_t attention(int dtype, const void* qkv, int64_t ld_qkv, void* out, int64_t ld_out, int B,
                      int K, int n_heads, int n_kv_heads, int head_dim, const Dev& dev) {
  if (B <= 0 || K <= 0) return cudaSuccess;
  if (dtype != kF32) return cudaErrorInvalidValue;   // bf16 runs attention_tc
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
