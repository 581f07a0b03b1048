// Folding a layer's norm parameters into the projections that read the
// normed rows (a reparameterisation: the layer computes the same function).
// For a norm y = n(x) * g + b feeding W (out = y W^T + c):
//   out = n(x) (W diag(g))^T + (c + W b)
// so W becomes W diag(g), the bias c + W b, and the norm's g, b become 1, 0.
// Layers whose gains are folded let the projections apply the norm's row
// scale in their epilogue instead of a separate normalisation pass.
#include "common.cuh"
#include "internal.h"

namespace adadsf {
namespace {

// c[n] += W[n, :] . b  (one warp per row of W, fp32 sums, one rounding)
template <typename T>
__global__ void fold_bias_kernel(const T* w, int N, int K, const T* b, T* c) {
  pdl_trigger();
  pdl_wait();
  const int n = blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
  const int lane = threadIdx.x & 31;
  if (n >= N) return;
  float s = 0.f;
  for (int k = lane; k < K; k += 32) s = fmaf(Elem<T>::to_f(w[(int64_t)n * K + k]), Elem<T>::to_f(b[k]), s);
  s = warp_sum(s);
  if (lane == 0) c[n] = Elem<T>::from_f(Elem<T>::to_f(c[n]) + s);
}

// W[n, k] *= g[k] in place (one rounding to the storage type)
template <typename T>
__global__ void fold_scale_kernel(T* w, int64_t N, int K, const T* g) {
  pdl_trigger();
  pdl_wait();
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= N * K) return;
  const int k = (int)(i % K);
  w[i] = Elem<T>::from_f(Elem<T>::to_f(w[i]) * Elem<T>::to_f(g[k]));
}

template <typename T>
__global__ void fill_kernel(T* v, int n, float value) {
  pdl_trigger();
  pdl_wait();
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) v[i] = Elem<T>::from_f(value);
}

template <typename T>
cudaError_t fold_one(T* w, int N, int K, const T* g, const T* b, T* bias, const Dev& dev) {
  cudaError_t e;
  if (b && bias) {
    e = launch_pdl(fold_bias_kernel<T>, dim3((N + 7) / 8), dim3(256), 0, dev.stream, (const T*)w, N, K, b, bias);
    if (e != cudaSuccess) return e;
  }
  const int64_t n = (int64_t)N * K;
  return launch_pdl(fold_scale_kernel<T>, dim3((unsigned)((n + 255) / 256)), dim3(256), 0, dev.stream, w,
                    (int64_t)N, K, g);
}

template <typename T>
cudaError_t reset_norm(T* g, T* b, int d, const Dev& dev) {
  const dim3 grid((d + 255) / 256);
  cudaError_t e = launch_pdl(fill_kernel<T>, grid, dim3(256), 0, dev.stream, g, d, 1.f);
  if (e != cudaSuccess || !b) return e;
  return launch_pdl(fill_kernel<T>, grid, dim3(256), 0, dev.stream, b, d, 0.f);
}

template <typename T>
cudaError_t fold_layer_t(bool neox, int d, int qkv, int F, T* w_qkv, T* b_qkv, T* w_up, T* b_up, T* w_gate,
                         T* g1, T* b1, T* g2, T* b2, const Dev& dev) {
  cudaError_t e;
  // first norm -> QKV (NeoX: its bias absorbs W_qkv b1)
  if ((e = fold_one<T>(w_qkv, qkv, d, g1, neox ? b1 : nullptr, b_qkv, dev)) != cudaSuccess) return e;
  // second norm -> MLP input projections (NeoX: up, its bias absorbs W_up b2;
  // Qwen: gate and up, no biases)
  if ((e = fold_one<T>(w_up, F, d, g2, neox ? b2 : nullptr, b_up, dev)) != cudaSuccess) return e;
  if (!neox && (e = fold_one<T>(w_gate, F, d, g2, nullptr, nullptr, dev)) != cudaSuccess) return e;
  if ((e = reset_norm<T>(g1, neox ? b1 : nullptr, d, dev)) != cudaSuccess) return e;
  return reset_norm<T>(g2, neox ? b2 : nullptr, d, dev);
}

}  // namespace

cudaError_t fold_layer_norms(int dtype, bool neox, int d, int qkv, int F, void* w_qkv, void* b_qkv, void* w_up,
                             void* b_up, void* w_gate, void* g1, void* b1, void* g2, void* b2, const Dev& dev) {
  if (dtype == kBF16)
    return fold_layer_t<bf16>(neox, d, qkv, F, (bf16*)w_qkv, (bf16*)b_qkv, (bf16*)w_up, (bf16*)b_up,
                              (bf16*)w_gate, (bf16*)g1, (bf16*)b1, (bf16*)g2, (bf16*)b2, dev);
  return fold_layer_t<float>(neox, d, qkv, F, (float*)w_qkv, (float*)b_qkv, (float*)w_up, (float*)b_up,
                             (float*)w_gate, (float*)g1, (float*)b1, (float*)g2, (float*)b2, dev);
}

}  // namespace adadsf
