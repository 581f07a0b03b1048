// Training-side pieces of AdaDSF (Sec. 3.5, Eqs. 9-11; Sec. 3.4's
// differentiable score pathway): the hidden-state alignment of one layer
// with its gradient, the output-distribution alignment (KL over the classes
// of an LM head), and the router's parameter gradient through the score gate
// of the gated variant. HBM- or latency-bound helpers around the forward;
// every reduction runs in a fixed order (results are bit-reproducible).
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace adadsf {
namespace {

constexpr int kRowThreadsT = 256;   // 8 warps, one row per warp step
constexpr int kMaxRowBlocks = 2048;

int row_blocks(int64_t n) {
  const int64_t want = (n + 7) / 8;
  return (int)(want < kMaxRowBlocks ? (want > 0 ? want : 1) : kMaxRowBlocks);
}

// Fixed-order sum of one double per block, added to acc[0]; acc[1] += count.
__global__ void sum_partials_kernel(const double* partials, int nblocks, int64_t count, double* acc) {
  pdl_trigger();
  pdl_wait();
  __shared__ double red[256];
  double s = 0;
  for (int i = threadIdx.x; i < nblocks; i += 256) s += partials[i];
  red[threadIdx.x] = s;
  __syncthreads();
  for (int o = 128; o > 0; o >>= 1) {
    if (threadIdx.x < o) red[threadIdx.x] += red[threadIdx.x + o];
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    acc[0] += red[0];
    acc[1] += (double)count;
  }
}

// Per-block fixed-order sum of the warps' per-row values.
__device__ __forceinline__ void block_partial(double mine, double* partials) {
  __shared__ double red[kRowThreadsT / 32];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  if (lane == 0) red[w] = mine;
  __syncthreads();
  if (threadIdx.x == 0) {
    double s = 0;
    for (int i = 0; i < kRowThreadsT / 32; ++i) s += red[i];
    partials[blockIdx.x] = s;
  }
}

// Eq. 9 per row (one warp): n = |softmax(hs) - softmax(hd)| over the d
// features, and, with grad, d n / d hs = p (r / n - p . r / n) (0 if n = 0),
// p = softmax(hs), r = p - softmax(hd). fp32, four passes over the rows.
template <typename T>
__global__ void __launch_bounds__(kRowThreadsT)
    align_hidden_kernel(const T* hs, const T* hd, int64_t n_rows, int d, float* grad, double* partials) {
  pdl_trigger();
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int64_t nw = (int64_t)gridDim.x * (kRowThreadsT / 32);
  double mine = 0;
  for (int64_t r = (int64_t)blockIdx.x * (kRowThreadsT / 32) + (threadIdx.x >> 5); r < n_rows; r += nw) {
    const T* a = hs + r * d;
    const T* b = hd + r * d;
    float ma = -INFINITY, mb = -INFINITY;
    for (int k = lane; k < d; k += 32) {
      ma = fmaxf(ma, Elem<T>::to_f(a[k]));
      mb = fmaxf(mb, Elem<T>::to_f(b[k]));
    }
    for (int o = 16; o > 0; o >>= 1) {
      ma = fmaxf(ma, __shfl_xor_sync(0xffffffffu, ma, o));
      mb = fmaxf(mb, __shfl_xor_sync(0xffffffffu, mb, o));
    }
    float za = 0.f, zb = 0.f;
    for (int k = lane; k < d; k += 32) {
      za += expf(Elem<T>::to_f(a[k]) - ma);
      zb += expf(Elem<T>::to_f(b[k]) - mb);
    }
    za = warp_sum(za);
    zb = warp_sum(zb);
    const float ia = 1.f / za, ib = 1.f / zb;
    float n2 = 0.f, pr = 0.f;
    for (int k = lane; k < d; k += 32) {
      const float p = expf(Elem<T>::to_f(a[k]) - ma) * ia;
      const float rr = p - expf(Elem<T>::to_f(b[k]) - mb) * ib;
      n2 = fmaf(rr, rr, n2);
      pr = fmaf(p, rr, pr);
    }
    n2 = warp_sum(n2);
    pr = warp_sum(pr);
    const float n = sqrtf(n2);
    mine += (double)n;   // identical on every lane; lane 0's copy is summed
    if (grad) {
      const float in = n > 0.f ? 1.f / n : 0.f;
      for (int k = lane; k < d; k += 32) {
        const float p = expf(Elem<T>::to_f(a[k]) - ma) * ia;
        const float rr = p - expf(Elem<T>::to_f(b[k]) - mb) * ib;
        grad[r * d + k] = p * (rr - pr) * in;
      }
    }
  }
  block_partial(mine, partials);
}

// Eq. 10 per row (one warp): KL(softmax(ld) || softmax(ls)) over n_cls
// classes, from fp32 logits.
__global__ void __launch_bounds__(kRowThreadsT)
    kl_rows_kernel(const float* ls, const float* ld, int64_t n_rows, int n_cls, double* partials) {
  pdl_trigger();
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int64_t nw = (int64_t)gridDim.x * (kRowThreadsT / 32);
  double mine = 0;
  for (int64_t r = (int64_t)blockIdx.x * (kRowThreadsT / 32) + (threadIdx.x >> 5); r < n_rows; r += nw) {
    const float* a = ls + r * n_cls;
    const float* b = ld + r * n_cls;
    float ma = -INFINITY, mb = -INFINITY;
    for (int k = lane; k < n_cls; k += 32) {
      ma = fmaxf(ma, a[k]);
      mb = fmaxf(mb, b[k]);
    }
    for (int o = 16; o > 0; o >>= 1) {
      ma = fmaxf(ma, __shfl_xor_sync(0xffffffffu, ma, o));
      mb = fmaxf(mb, __shfl_xor_sync(0xffffffffu, mb, o));
    }
    float za = 0.f, zb = 0.f;
    for (int k = lane; k < n_cls; k += 32) {
      za += expf(a[k] - ma);
      zb += expf(b[k] - mb);
    }
    za = warp_sum(za);
    zb = warp_sum(zb);
    // log P = logit - max - log Z
    const float la = ma + logf(za), lb = mb + logf(zb);
    float kl = 0.f;
    for (int k = lane; k < n_cls; k += 32) {
      const float lpb = b[k] - lb;
      kl = fmaf(expf(lpb), lpb - (a[k] - la), kl);
    }
    mine += (double)warp_sum(kl);
  }
  block_partial(mine, partials);
}

// Router gradient, part 1 (one warp per kept row m, flat row r = rows[m]):
// u = W1 x_r + b1 (h hidden units), s = w2 . SiLU(u) + b2, the gate's
// ds = sigmoid'(s) (G_r . delta_r) with delta_r = y_plain_r - x_r, and
// du = ds w2 SiLU'(u). Writes du [m][h], SiLU(u) [m][h] and ds [m].
template <typename T>
__global__ void __launch_bounds__(kRowThreadsT)
    router_bwd_rows_kernel(const T* x, const T* y_plain, const int32_t* rows, int64_t M, int d, int h,
                           const T* w1, const T* b1, const T* w2, const T* b2, const float* G, float* du,
                           float* su, float* ds_out) {
  pdl_trigger();
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int64_t nw = (int64_t)gridDim.x * (kRowThreadsT / 32);
  for (int64_t m = (int64_t)blockIdx.x * (kRowThreadsT / 32) + (threadIdx.x >> 5); m < M; m += nw) {
    const int64_t r = rows[m];
    const T* xr = x + r * d;
    const T* yr = y_plain + r * d;
    const float* gr = G + r * d;
    float gd = 0.f;
    for (int k = lane; k < d; k += 32) gd = fmaf(gr[k], Elem<T>::to_f(yr[k]) - Elem<T>::to_f(xr[k]), gd);
    gd = warp_sum(gd);
    float s = Elem<T>::to_f(b2[0]);
    for (int j = 0; j < h; ++j) {
      const T* wj = w1 + (int64_t)j * d;
      float dot = 0.f;
      for (int k = lane; k < d; k += 32) dot = fmaf(Elem<T>::to_f(wj[k]), Elem<T>::to_f(xr[k]), dot);
      const float u = warp_sum(dot) + Elem<T>::to_f(b1[j]);
      const float sg = 1.f / (1.f + expf(-u));
      s += Elem<T>::to_f(w2[j]) * u * sg;
      if (lane == 0) {
        su[m * h + j] = u * sg;
        du[m * h + j] = sg * (1.f + u * (1.f - sg));   // SiLU'(u), scaled by ds below
      }
    }
    const float sig = 1.f / (1.f + expf(-s));
    const float ds = sig * (1.f - sig) * gd;
    __syncwarp();
    for (int j = lane; j < h; j += 32) du[m * h + j] *= ds * Elem<T>::to_f(w2[j]);
    if (lane == 0) ds_out[m] = ds;
  }
}

// Router gradient, part 2: dW1[j][k] = sum_m du[m][j] x[rows[m]][k] (block b
// < nchunk: columns [128 b, 128 b + 128), 32 hidden units per thread);
// the last block: db1[j] = sum_m du[m][j], dw2[j] = sum_m ds[m] SiLU(u)[m][j],
// db2 = sum_m ds[m]. Rows summed in ascending m.
template <typename T>
__global__ void __launch_bounds__(256)
    router_bwd_reduce_kernel(const T* x, const int32_t* rows, int64_t M, int d, int h, const float* du,
                             const float* su, const float* ds, float* grad) {
  pdl_trigger();
  pdl_wait();
  const int nchunk = (d + 127) / 128;
  if ((int)blockIdx.x == nchunk) {
    for (int j = threadIdx.x; j < h; j += 256) {
      float gb1 = 0.f, gw2 = 0.f;
      for (int64_t m = 0; m < M; ++m) {
        gb1 += du[m * h + j];
        gw2 = fmaf(ds[m], su[m * h + j], gw2);
      }
      grad[(int64_t)h * d + j] = gb1;
      grad[(int64_t)h * d + h + j] = gw2;
    }
    if (threadIdx.x == 0) {
      float g = 0.f;
      for (int64_t m = 0; m < M; ++m) g += ds[m];
      grad[(int64_t)h * d + 2 * h] = g;
    }
    return;
  }
  const int k = (int)blockIdx.x * 128 + (threadIdx.x & 127);
  const int j0 = (threadIdx.x >> 7) * 32;   // 0 or 32 (h <= 64)
  float acc[32];
#pragma unroll
  for (int i = 0; i < 32; ++i) acc[i] = 0.f;
  __shared__ float sdu[32][64];
  __shared__ int64_t srow[32];
  for (int64_t m0 = 0; m0 < M; m0 += 32) {
    const int nm = (int)(M - m0 < 32 ? M - m0 : 32);
    __syncthreads();
    for (int i = threadIdx.x; i < 32 * 64; i += 256) {
      const int mm = i / 64, jj = i % 64;
      sdu[mm][jj] = (mm < nm && jj < h) ? du[(m0 + mm) * h + jj] : 0.f;
    }
    if (threadIdx.x < 32) srow[threadIdx.x] = threadIdx.x < nm ? (int64_t)rows[m0 + threadIdx.x] : 0;
    __syncthreads();
    if (k < d && j0 < h) {
      for (int mm = 0; mm < nm; ++mm) {
        const float xv = Elem<T>::to_f(x[srow[mm] * d + k]);
#pragma unroll
        for (int i = 0; i < 32; ++i) acc[i] = fmaf(sdu[mm][j0 + i], xv, acc[i]);
      }
    }
  }
  if (k < d)
    for (int i = 0; i < 32 && j0 + i < h; ++i) grad[(int64_t)(j0 + i) * d + k] = acc[i];
}

}  // namespace

int train_row_blocks(int64_t n) { return row_blocks(n); }

cudaError_t align_hidden(int dtype, const void* hs, const void* hd, int64_t n_rows, int d, float* grad,
                         double* partials, double* acc, const Dev& dev) {
  if (n_rows <= 0) return cudaSuccess;
  const int nb = row_blocks(n_rows);
  cudaError_t e;
  if (dtype == kBF16)
    e = launch_pdl(align_hidden_kernel<bf16>, dim3(nb), dim3(kRowThreadsT), 0, dev.stream,
                   static_cast<const bf16*>(hs), static_cast<const bf16*>(hd), n_rows, d, grad, partials);
  else
    e = launch_pdl(align_hidden_kernel<float>, dim3(nb), dim3(kRowThreadsT), 0, dev.stream,
                   static_cast<const float*>(hs), static_cast<const float*>(hd), n_rows, d, grad, partials);
  if (e != cudaSuccess) return e;
  return launch_pdl(sum_partials_kernel, dim3(1), dim3(256), 0, dev.stream, (const double*)partials, nb, n_rows,
                    acc);
}

cudaError_t kl_rows(const float* ls, const float* ld, int64_t n_rows, int n_cls, double* partials, double* acc,
                    const Dev& dev) {
  if (n_rows <= 0) return cudaSuccess;
  const int nb = row_blocks(n_rows);
  cudaError_t e = launch_pdl(kl_rows_kernel, dim3(nb), dim3(kRowThreadsT), 0, dev.stream, ls, ld, n_rows, n_cls,
                             partials);
  if (e != cudaSuccess) return e;
  return launch_pdl(sum_partials_kernel, dim3(1), dim3(256), 0, dev.stream, (const double*)partials, nb, n_rows,
                    acc);
}

cudaError_t router_backward(int dtype, const void* x, const void* y_plain, const int32_t* rows, int64_t M, int d,
                            int h, const void* w1, const void* b1, const void* w2, const void* b2, const float* G,
                            float* du, float* su, float* ds, float* grad, const Dev& dev) {
  if (h > 64) return cudaErrorInvalidValue;
  const int nchunk = (d + 127) / 128;
  if (M <= 0) return cudaMemsetAsync(grad, 0, sizeof(float) * ((size_t)h * d + 2 * h + 1), dev.stream);
  const int nb = row_blocks(M);
  cudaError_t e;
  if (dtype == kBF16) {
    e = launch_pdl(router_bwd_rows_kernel<bf16>, dim3(nb), dim3(kRowThreadsT), 0, dev.stream,
                   static_cast<const bf16*>(x), static_cast<const bf16*>(y_plain), rows, M, d, h,
                   static_cast<const bf16*>(w1), static_cast<const bf16*>(b1), static_cast<const bf16*>(w2),
                   static_cast<const bf16*>(b2), G, du, su, ds);
    if (e != cudaSuccess) return e;
    return launch_pdl(router_bwd_reduce_kernel<bf16>, dim3(nchunk + 1), dim3(256), 0, dev.stream,
                      static_cast<const bf16*>(x), rows, M, d, h, (const float*)du, (const float*)su,
                      (const float*)ds, grad);
  }
  e = launch_pdl(router_bwd_rows_kernel<float>, dim3(nb), dim3(kRowThreadsT), 0, dev.stream,
                 static_cast<const float*>(x), static_cast<const float*>(y_plain), rows, M, d, h,
                 static_cast<const float*>(w1), static_cast<const float*>(b1), static_cast<const float*>(w2),
                 static_cast<const float*>(b2), G, du, su, ds);
  if (e != cudaSuccess) return e;
  return launch_pdl(router_bwd_reduce_kernel<float>, dim3(nchunk + 1), dim3(256), 0, dev.stream,
                    static_cast<const float*>(x), rows, M, d, h, (const float*)du, (const float*)su,
                    (const float*)ds, grad);
}

}  // namespace adadsf
