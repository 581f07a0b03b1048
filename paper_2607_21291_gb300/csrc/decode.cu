// Autoregressive decode with a cache of kept tokens only. The paper (Sec.
// 3.4) defines the sparse forward over a whole sequence and is silent on
// generation; the reading implemented here: a generated token is kept at
// layer l when its router score beats the lowest score the layer kept in the
// prompt (the K-th largest of the Top-K, +inf when the layer kept nothing);
// a kept token attends to the layer's cached kept tokens and itself (rotary
// at original positions), gets the layer's residual delta, and its key and
// value join the cache; a skipped token bypasses the layer.
//
// Cache (one caller buffer, all device memory):
//   header   {T_cur, C_max, L, B} int32, padded to 256 bytes
//   lens     [L][B] int32     kept tokens cached per layer and sequence
//   thr      [L][B] fp32      keep thresholds
//   rope     [C_max][rot/2]   (cos, sin) fp32 pairs of every position
//   K, V     [L][B][Hkv][C_max][head_dim] each, storage dtype
// Every kernel reads positions and lengths from the cache, so a decode step
// has fixed launch arguments (capturable once in a CUDA graph).
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace adadsf {
namespace {

constexpr int kDecThreads = 128;        // 4 warps per attention CTA
constexpr int kMaxGroup = 16;           // query heads per key/value head

// ---------------------------------------------------------------- prefill -> cache
// K and V of the kept (packed) rows m = b K + j of one layer into the cache:
// row j of sequence b, every key/value head.
template <typename T>
__global__ void kv_fill_kernel(const T* qkv, int64_t ld, int q, int kvw, int B, int K, int hd,
                               int C_max, T* kc, T* vc) {
  pdl_trigger();
  pdl_wait();
  constexpr int V = Elem<T>::kVec;
  const int nvec = kvw / V;                       // 16-byte vectors of one row's keys
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (int64_t)B * K * nvec) return;
  const int64_t m = i / nvec;
  const int c = (int)(i % nvec) * V;              // feature within the kv width
  const int b = (int)(m / K), j = (int)(m % K);
  const int h = c / hd, e = c % hd;
  const int64_t dst = (((int64_t)b * (kvw / hd) + h) * C_max + j) * hd + e;
  *reinterpret_cast<uint4*>(kc + dst) = *reinterpret_cast<const uint4*>(qkv + m * ld + q + c);
  *reinterpret_cast<uint4*>(vc + dst) = *reinterpret_cast<const uint4*>(qkv + m * ld + q + kvw + c);
}

// Per sequence b: lens[b] = K and thr[b] = the lowest router score among its
// kept positions (+inf when K = 0). One block per sequence.
__global__ void kv_threshold_kernel(const float* scores, const int32_t* idx, int T, int K,
                                    int32_t* lens, float* thr) {
  pdl_trigger();
  pdl_wait();
  __shared__ float red[32];
  __shared__ int any_nan;
  const int b = blockIdx.x;
  if (threadIdx.x == 0) any_nan = 0;
  __syncthreads();
  float m = INFINITY;
  for (int j = threadIdx.x; j < K; j += blockDim.x) {
    const float s = scores[(int64_t)b * T + idx[(int64_t)b * K + j]];
    if (isnan(s)) any_nan = 1;   // a NaN was kept (fewer numbers than K): it is the minimum
    m = fminf(m, s);
  }
  for (int o = 16; o > 0; o >>= 1) m = fminf(m, __shfl_xor_sync(0xffffffffu, m, o));
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = m;
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int w = 1; w < (int)(blockDim.x >> 5); ++w) m = fminf(m, red[w]);
    lens[b] = K;
    thr[b] = any_nan ? NAN : m;
  }
}

__global__ void cache_header_kernel(int32_t* hdr, int T, int C_max, int L, int B) {
  pdl_trigger();
  pdl_wait();
  if (threadIdx.x == 0) {
    hdr[0] = T;
    hdr[1] = C_max;
    hdr[2] = L;
    hdr[3] = B;
  }
}

// ---------------------------------------------------------------- decode step
// Keep decision of the new token of every sequence at one layer, its
// position, and the packed-row map of the projections (rows[b] = b if kept,
// -1 if it bypasses the layer: the residual scatter then skips it).
__global__ void decode_decide_kernel(const float* scores, const float* thr, const int32_t* hdr, int B,
                                     int C_max, int32_t* rows, int32_t* pos, int32_t* kept_out, int* err) {
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  int t = hdr[0];
  // a cache not filled by a prefill of this shape, or no room left for the
  // position in its rotary table: flag it and stay in bounds
  if (hdr[1] != C_max || t < 0 || t >= C_max) {
    set_device_error(err, DEVERR_INDEX);
    t = t < 0 ? 0 : (t >= C_max ? C_max - 1 : t);
  }
  const bool keep = scores[b] > thr[b];   // a tie loses, NaN never wins
  rows[b] = keep ? b : -1;
  pos[b] = t;
  if (kept_out) kept_out[b] = keep ? 1 : 0;
}

// Attention of the new token of sequence b, query heads g0 .. g0 + G - 1 of
// key/value head h, over keys [lo, hi) of the n = lens[b] + 1 keys: the
// cached kept tokens, then the token itself (from qkv). One CTA per (split,
// kv head, sequence); each warp takes every 4th key with an online softmax
// per query head; the CTA's partial (max, sum, output) per head goes to
// part_ml / part_o for the combine step.
template <typename T>
__global__ void __launch_bounds__(kDecThreads)
    decode_attn_kernel(const T* qkv, int64_t ld, int q, int kvw, int Hq, int Hkv, int hd,
                       const T* kc, const T* vc, const int32_t* lens, int C_max, int nsplit,
                       float scale, float* part_o, float2* part_ml) {
  pdl_trigger();
  pdl_wait();
  const int s = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int G = Hq / Hkv;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int per = hd / 32;                        // features per lane (2 or 4)
  int len = lens[b];
  if (len < 0) len = 0;
  if (len > C_max) len = C_max;
  const int n = len + 1;
  const int lo = (int)((int64_t)s * n / nsplit), hi = (int)((int64_t)(s + 1) * n / nsplit);
  const T* qrow = qkv + (int64_t)b * ld;
  float qv[kMaxGroup][4];
  for (int g = 0; g < G; ++g)
    for (int i = 0; i < per; ++i)
      qv[g][i] = Elem<T>::to_f(qrow[(h * G + g) * hd + lane * per + i]) * scale;
  float mx[kMaxGroup], sm[kMaxGroup], acc[kMaxGroup][4];
  for (int g = 0; g < G; ++g) {
    mx[g] = -INFINITY;
    sm[g] = 0.f;
    for (int i = 0; i < per; ++i) acc[g][i] = 0.f;
  }
  const int64_t base = ((int64_t)b * Hkv + h) * C_max;
  for (int j = lo + warp; j < hi; j += 4) {
    const T* kr = j < len ? kc + (base + j) * hd : qrow + q + h * hd;
    const T* vr = j < len ? vc + (base + j) * hd : qrow + q + kvw + h * hd;
    float kf[4], vf[4];
    for (int i = 0; i < per; ++i) {
      kf[i] = Elem<T>::to_f(kr[lane * per + i]);
      vf[i] = Elem<T>::to_f(vr[lane * per + i]);
    }
    for (int g = 0; g < G; ++g) {
      float dot = 0.f;
      for (int i = 0; i < per; ++i) dot = fmaf(qv[g][i], kf[i], dot);
      dot = warp_sum(dot);
      const float mnew = fmaxf(mx[g], dot);
      const float corr = expf(mx[g] - mnew);
      const float pj = expf(dot - mnew);
      sm[g] = sm[g] * corr + pj;
      for (int i = 0; i < per; ++i) acc[g][i] = fmaf(acc[g][i], corr, pj * vf[i]);
      mx[g] = mnew;
    }
  }
  // merge the 4 warps' partials per head in shared memory
  __shared__ float s_ml[4][kMaxGroup][2];
  __shared__ float s_o[4][kMaxGroup][128];
  for (int g = 0; g < G; ++g) {
    if (lane == 0) {
      s_ml[warp][g][0] = mx[g];
      s_ml[warp][g][1] = sm[g];
    }
    for (int i = 0; i < per; ++i) s_o[warp][g][lane * per + i] = acc[g][i];
  }
  __syncthreads();
  for (int k = threadIdx.x; k < G * hd; k += kDecThreads) {
    const int g = k / hd, e = k % hd;
    float m = -INFINITY;
    for (int w = 0; w < 4; ++w) m = fmaxf(m, s_ml[w][g][0]);
    float l = 0.f, o = 0.f;
    if (m > -INFINITY) {
      for (int w = 0; w < 4; ++w) {
        const float c = expf(s_ml[w][g][0] - m);
        l += s_ml[w][g][1] * c;
        o += s_o[w][g][e] * c;
      }
    }
    const int64_t slot = ((int64_t)b * Hq + h * G + g) * nsplit + s;
    part_o[slot * hd + e] = o;
    if (e == 0) part_ml[slot] = make_float2(m, l);
  }
}

// out[b][head] = sum_s e^(m_s - m) o_s / sum_s e^(m_s - m) l_s over the splits.
template <typename T>
__global__ void decode_combine_kernel(const float* part_o, const float2* part_ml, int Hq, int hd,
                                      int nsplit, T* out, int64_t ld_out) {
  pdl_trigger();
  pdl_wait();
  const int hq = blockIdx.x, b = blockIdx.y;
  const int64_t slot0 = ((int64_t)b * Hq + hq) * nsplit;
  float m = -INFINITY;
  for (int s = 0; s < nsplit; ++s) m = fmaxf(m, part_ml[slot0 + s].x);
  for (int e = threadIdx.x; e < hd; e += blockDim.x) {
    float l = 0.f, o = 0.f;
    for (int s = 0; s < nsplit; ++s) {
      const float2 ml = part_ml[slot0 + s];
      if (ml.x == -INFINITY) continue;
      const float c = expf(ml.x - m);
      l += ml.y * c;
      o += part_o[(slot0 + s) * hd + e] * c;
    }
    out[(int64_t)b * ld_out + hq * hd + e] = Elem<T>::from_f(o / l);
  }
}

// The kept new tokens' keys and values join the layer's cache.
template <typename T>
__global__ void kv_append_kernel(const T* qkv, int64_t ld, int q, int kvw, int hd, int B,
                                 const int32_t* rows, int32_t* lens, int C_max, T* kc, T* vc,
                                 int* err) {
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x;
  if (rows[b] < 0) return;
  const int len = lens[b];
  if (len < 0 || len >= C_max) {
    if (threadIdx.x == 0) set_device_error(err, DEVERR_INDEX);
    return;
  }
  const int Hkv = kvw / hd;
  for (int c = threadIdx.x; c < kvw; c += blockDim.x) {
    const int h = c / hd, e = c % hd;
    const int64_t dst = (((int64_t)b * Hkv + h) * C_max + len) * hd + e;
    kc[dst] = qkv[(int64_t)b * ld + q + c];
    vc[dst] = qkv[(int64_t)b * ld + q + kvw + c];
  }
  __syncthreads();
  if (threadIdx.x == 0) lens[b] = len + 1;
}

__global__ void decode_advance_kernel(int32_t* hdr) {
  pdl_trigger();
  pdl_wait();
  if (threadIdx.x == 0) hdr[0] += 1;
}

}  // namespace

// ---------------------------------------------------------------- host side
int decode_splits(int B, int Hkv, int C_max, int num_sms) {
  const int units = B * Hkv;
  int s = (2 * num_sms + units - 1) / units;
  const int max_s = (C_max + 63) / 64;             // at least 64 keys a split
  if (s > max_s) s = max_s;
  if (s > 64) s = 64;
  return s < 1 ? 1 : s;
}

cudaError_t kv_fill(int dtype, const void* qkv, int64_t ld, int q, int kvw, int B, int K, int hd,
                    int C_max, void* kc, void* vc, const Dev& dev) {
  const int V = dtype == kBF16 ? 8 : 4;
  const int64_t n = (int64_t)B * K * (kvw / V);
  if (n <= 0) return cudaSuccess;
  const dim3 grid((unsigned)((n + 255) / 256));
  if (dtype == kBF16)
    return launch_pdl(kv_fill_kernel<bf16>, grid, dim3(256), 0, dev.stream, static_cast<const bf16*>(qkv), ld,
                      q, kvw, B, K, hd, C_max, static_cast<bf16*>(kc), static_cast<bf16*>(vc));
  return launch_pdl(kv_fill_kernel<float>, grid, dim3(256), 0, dev.stream, static_cast<const float*>(qkv), ld,
                    q, kvw, B, K, hd, C_max, static_cast<float*>(kc), static_cast<float*>(vc));
}

cudaError_t kv_threshold(const float* scores, const int32_t* idx, int B, int T, int K, int32_t* lens,
                         float* thr, const Dev& dev) {
  if (B <= 0) return cudaSuccess;
  return launch_pdl(kv_threshold_kernel, dim3(B), dim3(256), 0, dev.stream, scores, idx, T, K, lens, thr);
}

cudaError_t cache_header(int32_t* hdr, int T, int C_max, int L, int B, const Dev& dev) {
  return launch_pdl(cache_header_kernel, dim3(1), dim3(32), 0, dev.stream, hdr, T, C_max, L, B);
}

cudaError_t decode_decide(const float* scores, const float* thr, const int32_t* hdr, int B, int C_max,
                          int32_t* rows, int32_t* pos, int32_t* kept_out, const Dev& dev) {
  return launch_pdl(decode_decide_kernel, dim3((B + 127) / 128), dim3(128), 0, dev.stream, scores, thr, hdr, B,
                    C_max, rows, pos, kept_out, dev.err);
}

cudaError_t decode_attention(int dtype, const void* qkv, int64_t ld, int Hq, int Hkv, int hd, const void* kc,
                             const void* vc, const int32_t* lens, int C_max, int B, float* part_o,
                             float2* part_ml, void* out, int64_t ld_out, const Dev& dev) {
  if (B <= 0) return cudaSuccess;
  if (Hq % Hkv != 0 || Hq / Hkv > kMaxGroup || (hd != 64 && hd != 128)) return cudaErrorInvalidValue;
  const int q = Hq * hd, kvw = Hkv * hd;
  const int ns = decode_splits(B, Hkv, C_max, dev.num_sms);
  const float scale = 1.f / sqrtf((float)hd);
  const dim3 grid(ns, Hkv, B);
  cudaError_t e;
  if (dtype == kBF16)
    e = launch_pdl(decode_attn_kernel<bf16>, grid, dim3(kDecThreads), 0, dev.stream,
                   static_cast<const bf16*>(qkv), ld, q, kvw, Hq, Hkv, hd, static_cast<const bf16*>(kc),
                   static_cast<const bf16*>(vc), lens, C_max, ns, scale, part_o, part_ml);
  else
    e = launch_pdl(decode_attn_kernel<float>, grid, dim3(kDecThreads), 0, dev.stream,
                   static_cast<const float*>(qkv), ld, q, kvw, Hq, Hkv, hd, static_cast<const float*>(kc),
                   static_cast<const float*>(vc), lens, C_max, ns, scale, part_o, part_ml);
  if (e != cudaSuccess) return e;
  if (dtype == kBF16)
    return launch_pdl(decode_combine_kernel<bf16>, dim3(Hq, B), dim3(128), 0, dev.stream, part_o, part_ml, Hq,
                      hd, ns, static_cast<bf16*>(out), ld_out);
  return launch_pdl(decode_combine_kernel<float>, dim3(Hq, B), dim3(128), 0, dev.stream, part_o, part_ml, Hq, hd,
                    ns, static_cast<float*>(out), ld_out);
}

cudaError_t kv_append(int dtype, const void* qkv, int64_t ld, int q, int kvw, int hd, int B, const int32_t* rows,
                      int32_t* lens, int C_max, void* kc, void* vc, const Dev& dev) {
  if (B <= 0) return cudaSuccess;
  if (dtype == kBF16)
    return launch_pdl(kv_append_kernel<bf16>, dim3(B), dim3(256), 0, dev.stream, static_cast<const bf16*>(qkv),
                      ld, q, kvw, hd, B, rows, lens, C_max, static_cast<bf16*>(kc), static_cast<bf16*>(vc),
                      dev.err);
  return launch_pdl(kv_append_kernel<float>, dim3(B), dim3(256), 0, dev.stream, static_cast<const float*>(qkv),
                    ld, q, kvw, hd, B, rows, lens, C_max, static_cast<float*>(kc), static_cast<float*>(vc),
                    dev.err);
}

cudaError_t decode_advance(int32_t* hdr, const Dev& dev) {
  return launch_pdl(decode_advance_kernel, dim3(1), dim3(32), 0, dev.stream, hdr);
}

}  // namespace adadsf
