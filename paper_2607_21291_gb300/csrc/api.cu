// C ABI of the depth-sparse forward (declared in include/adadsf.h): argument
// validation, workspace carving, the per-layer launch sequence and the host
// retention allocation. No entry point allocates device memory or
// synchronises a stream except adadsf_sync_check.
#include <math.h>
#include <stdarg.h>
#include <stdio.h>

#include <map>
#include <mutex>
#include <string>
#include <utility>
#include <vector>

#include "adadsf.h"
#include "internal.h"

using namespace adadsf;

namespace {

thread_local std::string g_last_error;

adadsf_status fail(adadsf_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return s;
}

adadsf_status cuda_fail(cudaError_t e, const char* what) {
  return fail(ADADSF_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

#define CUDA_TRY(expr, what)                    \
  do {                                          \
    cudaError_t e_ = (expr);                    \
    if (e_ != cudaSuccess) return cuda_fail(e_, what); \
  } while (0)

#define TRY(expr)                               \
  do {                                          \
    adadsf_status s_ = (expr);                  \
    if (s_ != ADADSF_OK) return s_;             \
  } while (0)

constexpr size_t kErrBytes = 256;

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int elem_size(int dtype) { return dtype == kBF16 ? 2 : 4; }

adadsf_status device_info(Dev* dev, void* stream, void* ws) {
  int device = 0;
  CUDA_TRY(cudaGetDevice(&device), "cudaGetDevice");
  static int sms[64] = {0};
  if (device >= 64) return fail(ADADSF_ERR_UNSUPPORTED, "device ordinal %d >= 64", device);
  if (!sms[device]) {
    int n = 0;
    CUDA_TRY(cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, device),
             "cudaDeviceGetAttribute");
    sms[device] = n;
  }
  dev->num_sms = sms[device];
  dev->stream = static_cast<cudaStream_t>(stream);
  dev->err = static_cast<int*>(ws);
  return ADADSF_OK;
}

adadsf_status check_cfg(const adadsf_model_cfg* c) {
  if (!c) return fail(ADADSF_ERR_INVALID_ARG, "cfg is NULL");
  if (c->dtype != ADADSF_F32 && c->dtype != ADADSF_BF16)
    return fail(ADADSF_ERR_INVALID_ARG, "dtype %d is neither ADADSF_F32 nor ADADSF_BF16", c->dtype);
  if (c->arch != ADADSF_ARCH_NEOX && c->arch != ADADSF_ARCH_QWEN)
    return fail(ADADSF_ERR_INVALID_ARG, "arch %d unknown", c->arch);
  const int vec = c->dtype == ADADSF_BF16 ? 8 : 4;
  if (c->d <= 0 || c->d % 64 != 0)
    return fail(ADADSF_ERR_UNSUPPORTED, "d=%d must be a positive multiple of 64", c->d);
  if (c->d > 16 * 32 * vec)
    return fail(ADADSF_ERR_UNSUPPORTED, "d=%d exceeds %d for this dtype", c->d, 16 * 32 * vec);
  if (c->head_dim != 64 && c->head_dim != 128)
    return fail(ADADSF_ERR_UNSUPPORTED, "head_dim=%d must be 64 or 128", c->head_dim);
  if (c->n_heads <= 0 || c->n_kv_heads <= 0 || c->n_heads % c->n_kv_heads != 0)
    return fail(ADADSF_ERR_INVALID_ARG, "n_heads=%d must be a positive multiple of n_kv_heads=%d",
                c->n_heads, c->n_kv_heads);
  if (c->ffn <= 0 || c->ffn % 64 != 0)
    return fail(ADADSF_ERR_UNSUPPORTED, "ffn=%d must be a positive multiple of 64", c->ffn);
  if (c->dtype == ADADSF_BF16 && c->router_hidden != 64)
    return fail(ADADSF_ERR_UNSUPPORTED, "bf16 router_hidden=%d must be 64", c->router_hidden);
  if (c->router_hidden <= 0 || c->router_hidden > 1024)
    return fail(ADADSF_ERR_INVALID_ARG, "router_hidden=%d out of range", c->router_hidden);
  if (c->rotary_dim < 0 || c->rotary_dim > c->head_dim || c->rotary_dim % 2 != 0)
    return fail(ADADSF_ERR_INVALID_ARG, "rotary_dim=%d must be even and <= head_dim", c->rotary_dim);
  if (!(c->norm_eps > 0.f) || !(c->rope_theta > 0.f))
    return fail(ADADSF_ERR_INVALID_ARG, "norm_eps and rope_theta must be positive");
  if ((unsigned)c->flags & ~(unsigned)(ADADSF_FLAG_GATE_SIGMOID | ADADSF_FLAG_FOLDED_NORMS | ADADSF_FLAG_GATHERED_QKV))
    return fail(ADADSF_ERR_UNSUPPORTED, "flags 0x%x has unknown bits", (unsigned)c->flags);
  return ADADSF_OK;
}

bool gated(const adadsf_model_cfg* c) { return ((unsigned)c->flags & ADADSF_FLAG_GATE_SIGMOID) != 0; }
bool folded(const adadsf_model_cfg* c) { return ((unsigned)c->flags & ADADSF_FLAG_FOLDED_NORMS) != 0; }
bool gathered_qkv(const adadsf_model_cfg* c) {
  return folded(c) && ((unsigned)c->flags & ADADSF_FLAG_GATHERED_QKV) != 0;
}

adadsf_status check_shape(int B, int T, int K) {
  if (B < 0 || T <= 0 || K < 0 || K > T)
    return fail(ADADSF_ERR_INVALID_ARG, "need B >= 0, T > 0, 0 <= K <= T (B=%d T=%d K=%d)", B, T, K);
  if (T > 16384) return fail(ADADSF_ERR_UNSUPPORTED, "T=%d exceeds 16384", T);
  if ((int64_t)B * T > (int64_t)1 << 30) return fail(ADADSF_ERR_UNSUPPORTED, "B*T too large");
  return ADADSF_OK;
}

adadsf_status check_ws(void* ws, size_t ws_bytes, size_t need) {
  if (!ws) return fail(ADADSF_ERR_INVALID_ARG, "workspace is NULL");
  if (reinterpret_cast<uintptr_t>(ws) & 255u)
    return fail(ADADSF_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
  if (ws_bytes < need)
    return fail(ADADSF_ERR_WORKSPACE_TOO_SMALL, "workspace has %zu bytes, needs %zu", ws_bytes, need);
  return ADADSF_OK;
}

// ---------------------------------------------------------------- per-launch timing
struct Profiler {
  std::mutex mu;
  bool on = false;
  int cap = 0;
  std::vector<cudaEvent_t> ev;   // two per record
  std::vector<adadsf_launch_record> recs;
  std::vector<int> rec_err;       // cudaEventRecord status of each record
};
Profiler g_prof;

// Runs f() (which enqueues one kernel or copy on dev.stream); while profiling
// is on and the stream is not being captured, brackets it with events.
template <typename F>
adadsf_status launch(const Dev& dev, int kind, bool dense, double flops, double bytes, F&& f) {
  cudaEvent_t a = nullptr, b = nullptr;
  size_t slot = 0;
  if (g_prof.on) {
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(dev.stream, &cs) == cudaSuccess && cs == cudaStreamCaptureStatusNone) {
      std::lock_guard<std::mutex> lk(g_prof.mu);
      const size_t i = g_prof.recs.size();
      if ((int)i < g_prof.cap) {
        a = g_prof.ev[2 * i];
        b = g_prof.ev[2 * i + 1];
        g_prof.recs.push_back({kind, dense ? 1 : 0, 0.0, flops, bytes});
        g_prof.rec_err.push_back(0);
        slot = i;
      }
    }
  }
  const cudaError_t ea = a ? cudaEventRecord(a, dev.stream) : cudaSuccess;
  const adadsf_status st = f();
  const cudaError_t eb = b ? cudaEventRecord(b, dev.stream) : cudaSuccess;
  if (ea != cudaSuccess || eb != cudaSuccess) {
    std::lock_guard<std::mutex> lk(g_prof.mu);
    g_prof.rec_err[slot] = ea != cudaSuccess ? (int)ea : (int)eb;
  }
  return st;
}

#define NEED_PTR(p, name)                                                             \
  do {                                                                                \
    if (!(p)) return fail(ADADSF_ERR_INVALID_ARG, "%s is NULL", name);                \
    if (!aligned16(p)) return fail(ADADSF_ERR_INVALID_ARG, "%s is not 16-byte aligned", name); \
  } while (0)

adadsf_status check_layer_weights(const adadsf_model_cfg* c, const adadsf_layer_weights* w,
                                  bool need_router) {
  if (!w) return fail(ADADSF_ERR_INVALID_ARG, "layer weights are NULL");
  if (need_router) {
    NEED_PTR(w->router_w1, "router_w1");
    NEED_PTR(w->router_b1, "router_b1");
    NEED_PTR(w->router_w2, "router_w2");
    if (!w->router_b2) return fail(ADADSF_ERR_INVALID_ARG, "router_b2 is NULL");
  }
  NEED_PTR(w->ln1_w, "ln1_w");
  NEED_PTR(w->ln2_w, "ln2_w");
  NEED_PTR(w->w_qkv, "w_qkv");
  NEED_PTR(w->b_qkv, "b_qkv");
  NEED_PTR(w->w_o, "w_o");
  NEED_PTR(w->w_up, "w_up");
  NEED_PTR(w->w_down, "w_down");
  if (c->arch == ADADSF_ARCH_NEOX) {
    NEED_PTR(w->ln1_b, "ln1_b");
    NEED_PTR(w->ln2_b, "ln2_b");
    NEED_PTR(w->b_o, "b_o");
    NEED_PTR(w->b_up, "b_up");
    NEED_PTR(w->b_down, "b_down");
  } else {
    NEED_PTR(w->w_gate, "w_gate");
  }
  return ADADSF_OK;
}

// ---------------------------------------------------------------- workspace layout
struct Carver {
  size_t cur = 0;
  size_t take(size_t bytes) {
    const size_t o = cur;
    cur = align256(cur + bytes);
    return o;
  }
};

struct LayerSlots {
  size_t scores, idx, rows, n1, n2, qkv, vt, attn, ao, act, split, rsel, sq, tsq;
};

void carve_layer(const adadsf_model_cfg* c, int B, int T, int K, Carver& cv, LayerSlots& s) {
  const size_t es = elem_size(c->dtype);
  const size_t M = (size_t)B * K;
  const size_t q = (size_t)c->n_heads * c->head_dim, kv = (size_t)c->n_kv_heads * c->head_dim;
  s.scores = cv.take((size_t)B * T * 4);
  s.idx = cv.take(M * 4);
  s.rows = cv.take(M * 4);
  s.n1 = cv.take(M * c->d * es);
  s.n2 = c->arch == ADADSF_ARCH_NEOX ? cv.take(M * c->d * es) : 0;
  s.qkv = cv.take(M * (q + 2 * kv) * es);
  // value heads transposed for the tensor-core attention: [B][Hkv][hd][vt_pad(K)]
  s.vt = c->dtype == ADADSF_BF16 ? cv.take((size_t)B * kv * vt_pad(K) * es) : 0;
  s.attn = cv.take(M * q * es);
  s.ao = cv.take(M * c->d * es);
  s.act = cv.take(M * c->ffn * es);
  // fp32 partial tiles of projections split along K (tensor-core path)
  s.split = c->dtype == ADADSF_BF16 ? cv.take(gemm_split_scratch_bytes()) : 0;
  // router partial tiles (tensor-core path; its counters sit in the
  // workspace's synchronisation area)
  s.rsel = c->dtype == ADADSF_BF16 ? cv.take(router_partial_bytes()) : 0;
  // per-chunk sums of squares of h (Qwen, bf16, folded norms: the second
  // RMSNorm applied in the gate / up epilogue)
  s.sq = c->dtype == ADADSF_BF16 && c->arch == ADADSF_ARCH_QWEN ? cv.take(M * (c->d / 32) * 4) : 0;
  // every token's sum of squares from the router (Qwen, bf16, folded norms:
  // the first RMSNorm applied in the QKV epilogue)
  s.tsq = c->dtype == ADADSF_BF16 && c->arch == ADADSF_ARCH_QWEN && gathered_qkv(c) ? cv.take((size_t)B * T * 4) : 0;
}

size_t rope_bytes(const adadsf_model_cfg* c, int T) { return (size_t)T * (c->rotary_dim / 2) * 8; }

template <typename T>
T* at(void* ws, size_t off) {
  return reinterpret_cast<T*>(static_cast<char*>(ws) + off);
}

// ---------------------------------------------------------------- one layer
struct LayerBufs {
  float* scores;
  int32_t* idx;
  int32_t* rows;
  const float2* rope;
  void *n1, *n2, *qkv, *vt, *attn, *ao, *act;
  float* split;   // null on the fp32 path
  int* sync;       // the workspace's synchronisation area
  float* rpart;    // router partial tiles, null on the fp32 path
  float* sq = nullptr;        // [M][d/32] chunk sums of squares of h (folded second RMSNorm)
  float* tsq = nullptr;       // [B T] sums of squares of the layer input rows (folded first RMSNorm)
  float4* cospart = nullptr;  // [B T][d/32] Eq. 4 partials from the down epilogue (dense, bf16)
};

adadsf_status run_linear(int dtype, const GemmArgs& g, const Dev& dev, const char* what) {
  cudaError_t e = dtype == kBF16 ? gemm_bf16(g, dev) : gemm_f32(g, dev);
  if (e != cudaSuccess) return cuda_fail(e, what);
  return ADADSF_OK;
}

GemmArgs linear_args(const void* A, int64_t lda, const void* W, int64_t M, int N, int K) {
  GemmArgs g;
  g.A = A; g.lda = lda; g.W = W; g.ldw = K;
  g.M = M; g.N = N; g.K = K;
  return g;
}

#define CALL(expr, what)                 \
  [&]() -> adadsf_status {               \
    cudaError_t e_ = (expr);             \
    if (e_ != cudaSuccess) return cuda_fail(e_, what); \
    return ADADSF_OK;                    \
  }

// Prefill into a decode cache: the layer's kept keys / values, kept counts
// and keep thresholds (see decode.cu).
struct CacheSink {
  void *kc, *vc;
  int32_t* lens;   // [B]
  float* thr;      // [B]
  int C_max;
};

// One decode step of a layer: B new tokens (one per sequence, T = K = 1).
struct DecodeCtx {
  const float* thr;      // [B] this layer's thresholds
  const int32_t* hdr;    // cache header (current position)
  int32_t* lens;         // [B] this layer's cached counts
  void *kc, *vc;         // this layer's cache
  int C_max;
  int32_t* rows;         // [B] b if kept, -1 if the token bypasses the layer
  int32_t* pos;          // [B] the token's position
  float* part_o;         // split-attention partials
  float2* part_ml;
  int32_t* kept_out;     // [B] or null
  // A second stream for the router and the keep decision, which need only
  // the layer input, so they run beside the norm and the QKV projection;
  // joined before the cache append (null: everything on one stream).
  cudaStream_t side = nullptr;
  cudaEvent_t fork = nullptr, join = nullptr;
};

// The second stream and the two events of decode steps on the caller's
// stream `main` (of the current device), made once per such stream (not
// while `main` is being captured into a graph: the step then runs on one
// stream). Keyed by the caller's stream, so that steps enqueued on different
// streams from different host threads never share the fork and join events.
// False when they are not available.
bool decode_side_stream(cudaStream_t main, cudaStream_t* side, cudaEvent_t* fork, cudaEvent_t* join) {
  struct Side {
    cudaStream_t s = nullptr;
    cudaEvent_t f = nullptr, j = nullptr;
  };
  static std::mutex mu;
  static std::map<std::pair<int, cudaStream_t>, Side> by_stream;
  int device = 0;
  if (cudaGetDevice(&device) != cudaSuccess) return false;
  std::lock_guard<std::mutex> lk(mu);
  const auto key = std::make_pair(device, main);
  auto it = by_stream.find(key);
  if (it == by_stream.end()) {
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(main, &cs) != cudaSuccess || cs != cudaStreamCaptureStatusNone) return false;
    Side sd;
    if (cudaStreamCreateWithFlags(&sd.s, cudaStreamNonBlocking) != cudaSuccess) return false;
    if (cudaEventCreateWithFlags(&sd.f, cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&sd.j, cudaEventDisableTiming) != cudaSuccess) {
      cudaGetLastError();
      return false;
    }
    it = by_stream.emplace(key, sd).first;
  }
  *side = it->second.s;
  *fork = it->second.f;
  *join = it->second.j;
  return true;
}

// Sec. 3.4: router -> Top-K -> gather + norm -> block on the packed rows ->
// residual delta scattered back into x. K == T skips router and Top-K.
// sink: also fill a decode cache (prefill). dec: a decode step instead.
adadsf_status layer_impl(const adadsf_model_cfg* c, const adadsf_layer_weights* w, void* x, int B,
                         int T, int K, const LayerBufs& lb, bool want_idx, const Dev& dev,
                         const CacheSink* sink = nullptr, const DecodeCtx* dec = nullptr) {
  if (K == 0 || B == 0) {
    // a layer that keeps nothing: an empty cache that keeps nothing either
    if (sink && B > 0)
      TRY(launch(dev, ADADSF_KERNEL_KV_CACHE, false, 0, 8.0 * B,
                 CALL(kv_threshold(lb.scores, lb.idx, B, T, 0, sink->lens, sink->thr, dev), "cache thresholds")));
    return ADADSF_OK;
  }
  const bool dense = K == T && !dec;
  const bool gate = gated(c);
  const int dt = c->dtype, d = c->d;
  const double es = elem_size(dt);
  const int64_t M = (int64_t)B * K;
  const int64_t BT = (int64_t)B * T;
  const int q = c->n_heads * c->head_dim, kv = c->n_kv_heads * c->head_dim;
  const int qkv_dim = q + 2 * kv;
  const int F = c->ffn;
  const bool neox = c->arch == ADADSF_ARCH_NEOX;
  const bool tc = dt == kBF16;   // dense contractions on tensor cores
  const double Md = (double)M * d;
  const int32_t* rows = nullptr;
  const int32_t* pos = nullptr;

  // decode on two streams: the router and the keep decision on the side
  // stream (from the layer input x), the norm and QKV on the main one
  const bool forked = dec && dec->side;
  Dev sdev = dev;
  if (forked) {
    sdev.stream = dec->side;
    CUDA_TRY(cudaEventRecord(dec->fork, dev.stream), "fork the router stream");
    CUDA_TRY(cudaStreamWaitEvent(dec->side, dec->fork, 0), "fork the router stream");
  }
  // a4 inside the QKV projection (opt-in; bf16 Qwen layers with folded gains
  // that take the Top-K path): the router also leaves each token's sum of
  // squares, the projection loads the kept rows of x by row gathers, and its
  // epilogue scales each row by 1 / rms before the bias and rotary.
  const bool fuse1 = tc && !dec && !dense && !neox && gathered_qkv(c) && lb.tsq && M > 32LL * dev.num_sms;
  if (!dense || gate || sink) {
    const double rf = 2.0 * BT * c->router_hidden * d;
    const double rb = (double)BT * d * es + (double)c->router_hidden * d * es + BT * 4.0;
    // a2: router scores of every token (bf16: tensor cores, tiles split
    // along d when there are few of them); the gated variant also needs
    // them when every token is kept
    TRY(launch(sdev, ADADSF_KERNEL_ROUTER, false, rf, rb,
               CALL(tc ? router_tc(x, BT, d, w->router_w1, w->router_b1, w->router_w2, w->router_b2,
                                   lb.scores, fuse1 ? lb.tsq : nullptr, lb.sync, lb.rpart, sdev)
                       : router_f32(static_cast<const float*>(x), BT, d, c->router_hidden,
                                    static_cast<const float*>(w->router_w1),
                                    static_cast<const float*>(w->router_b1),
                                    static_cast<const float*>(w->router_w2),
                                    static_cast<const float*>(w->router_b2), lb.scores, sdev),
                    "router")));
  }
  if (dec) {
    // decode: keep decision of each new token and the norms of all B rows
    // (a bypassing token's block output is computed and dropped: the
    // projections stream their weights once either way)
    if (forked) {
      TRY(launch(sdev, ADADSF_KERNEL_DECIDE, false, 0, 16.0 * B,
                 CALL(decode_decide(lb.scores, dec->thr, dec->hdr, B, dec->C_max, dec->rows, dec->pos,
                                    dec->kept_out, sdev),
                      "keep decision")));
      CUDA_TRY(cudaEventRecord(dec->join, dec->side), "join the router stream");
      TRY(launch(dev, ADADSF_KERNEL_GATHER_NORM, false, 0, Md * es * (neox ? 3 : 2),
                 CALL(gather_norm(dt, x, nullptr, M, d, !neox, w->ln1_w, w->ln1_b, w->ln2_w, w->ln2_b,
                                  c->norm_eps, lb.n1, neox ? lb.n2 : nullptr, dev),
                      "norm")));
    } else {
      TRY(launch(dev, ADADSF_KERNEL_GATHER_NORM, false, 0, Md * es * (neox ? 3 : 2) + 16.0 * B,
                 CALL(decide_norm(dt, x, B, d, !neox, w->ln1_w, w->ln1_b, w->ln2_w, w->ln2_b, c->norm_eps,
                                  lb.n1, neox ? lb.n2 : nullptr, lb.scores, dec->thr, dec->hdr, dec->C_max,
                                  dec->rows, dec->pos, dec->kept_out, dev),
                      "keep decision + norm")));
    }
    rows = dec->rows;
    pos = dec->pos;
  } else if (!dense) {
    if (M <= 32LL * dev.num_sms) {
      // a3 + a4: Top-K of each sequence fused with the gather of the kept rows
      // and their norms (NeoX: LN1 and LN2 of the same row). Every block
      // repeats its sequence's selection: worth it while a launch less
      // outweighs that (up to about one row per warp on four blocks per SM).
      TRY(launch(dev, ADADSF_KERNEL_TOPK_GATHER_NORM, false, 0,
                 BT * 4.0 + M * 8.0 + Md * es * (neox ? 3 : 2),
                 CALL(select_gather_norm(dt, lb.scores, B, T, K, x, d, !neox, w->ln1_w, w->ln1_b,
                                         w->ln2_w, w->ln2_b, c->norm_eps, lb.n1,
                                         neox ? lb.n2 : nullptr, lb.idx, lb.rows, dev),
                      "top-k + gather + norm")));
    } else {
      TRY(launch(dev, ADADSF_KERNEL_TOPK, false, 0, BT * 4.0 + M * 8.0,
                 CALL(topk(lb.scores, B, T, K, lb.idx, lb.rows, dev), "top-k")));
      // a4: gather the kept rows and normalise them (NeoX: LN1 and LN2)
      if (!fuse1)
        TRY(launch(dev, ADADSF_KERNEL_GATHER_NORM, false, 0, Md * es * (neox ? 3 : 2),
                   CALL(gather_norm(dt, x, lb.rows, M, d, !neox, w->ln1_w, w->ln1_b, w->ln2_w,
                                    w->ln2_b, c->norm_eps, lb.n1, neox ? lb.n2 : nullptr, dev),
                        "gather+norm")));
    }
    rows = lb.rows;
    pos = lb.idx;
  } else {
    if (want_idx || sink)
      TRY(launch(dev, ADADSF_KERNEL_POSITIONS, false, 0, M * 4.0,
                 CALL(iota_positions(lb.idx, B, K, dev), "positions")));
    // a4: normalise every row (NeoX: LN1 and LN2 of the same row).
    TRY(launch(dev, ADADSF_KERNEL_GATHER_NORM, false, 0, Md * es * (neox ? 3 : 2),
               CALL(gather_norm(dt, x, nullptr, M, d, !neox, w->ln1_w, w->ln1_b, w->ln2_w,
                                w->ln2_b, c->norm_eps, lb.n1, neox ? lb.n2 : nullptr, dev),
                    "norm")));
  }
  // a5: QKV projection (+bias), rotary at the original positions.
  // On the tensor-core path the rotation is fused into the QKV epilogue, and
  // for GPT-NeoX (parallel residual) the MLP up projection of the second
  // norm shares the launch (a8).
  const int half = c->rotary_dim / 2;
  // (not in a decode step: with a few rows the projection runs split along K,
  // which rotary tiles of halves above 16 features rule out; a separate pass
  // rotates the few rows instead)
  const bool fuse_rope = tc && !dec && (half == 4 || half == 8 || half == 16 || (half > 0 && half % 32 == 0));
  const bool neox_tc = neox && tc;
  {
    GemmArgs g = linear_args(fuse1 ? x : lb.n1, d, w->w_qkv, M, qkv_dim, d);
    g.scratch = lb.split;
    g.scratch_bytes = lb.split ? gemm_split_scratch_bytes() : 0;
    if (fuse1) {
      g.a_gather = lb.rows;
      g.a_gather_rows = BT;
      g.epi.nrm_psum = lb.tsq;
      g.epi.nrm_rows = lb.rows;
      g.epi.nrm_nps = 1;
      g.epi.nrm_d = d;
      g.epi.nrm_eps = c->norm_eps;
    }
    g.epi.bias = w->b_qkv;
    g.epi.out = lb.qkv;
    g.epi.ld_out = qkv_dim;
    if (fuse_rope) {
      g.epi.rope_tab = lb.rope;
      g.epi.rope_pos = pos;
      g.epi.rope_T = T;
      g.epi.rope_half = half;
      g.epi.rope_hd = c->head_dim;
      g.epi.rope_cols = (c->n_heads + c->n_kv_heads) * c->head_dim;
    }
    if (tc && !dec) {
      g.epi.vt = lb.vt;
      g.epi.vt_seq = K;
      g.epi.vt_pad = vt_pad(K);
      g.epi.vt_col0 = q + kv;
      g.epi.vt_hd = c->head_dim;
      g.epi.vt_hkv = c->n_kv_heads;
    }
    if (neox_tc) {
      // act = GELU(LN2 x W_up^T + b_up), grouped with the QKV tiles (first:
      // its GELU epilogue is the costlier)
      GemmArgs u = linear_args(lb.n2, d, w->w_up, M, F, d);
      u.epi.bias = w->b_up;
      u.epi.act = ACT_GELU;
      u.epi.out = lb.act;
      u.epi.ld_out = F;
      TRY(launch(dev, ADADSF_KERNEL_GEMM_QKV_UP, true, 2.0 * M * ((double)qkv_dim + F) * d,
                 (2.0 * Md + ((double)qkv_dim + F) * d + (double)M * (qkv_dim + F)) * es,
                 CALL(gemm_bf16_grouped(u, g, dev), "qkv + mlp up projections")));
    } else {
      TRY(launch(dev, ADADSF_KERNEL_GEMM_QKV, tc, 2.0 * M * qkv_dim * d,
                 (Md + (double)qkv_dim * d + (double)M * qkv_dim) * es,
                 [&] { return run_linear(dt, g, dev, "qkv projection"); }));
    }
  }
  if (c->rotary_dim > 0 && !fuse_rope && !dec)
    TRY(launch(dev, ADADSF_KERNEL_ROPE, false, 0,
               2.0 * M * (c->n_heads + c->n_kv_heads) * c->rotary_dim * es,
               CALL(rope_apply(dt, lb.qkv, M, qkv_dim, c->n_heads, c->n_kv_heads, c->head_dim,
                               c->rotary_dim, pos, T, lb.rope, dev),
                    "rotary")));
  if (dec) {
    if (forked) CUDA_TRY(cudaStreamWaitEvent(dev.stream, dec->join, 0), "join the router stream");
    // a5' + a6 (decode): rotary of the new rows fused with the cache append
    // (a kept token's rotated key and value join the cache), then each new
    // token attends to its layer's cached kept tokens (itself included when kept)
    TRY(launch(dev, ADADSF_KERNEL_KV_CACHE, false, 0,
               2.0 * M * (c->n_heads + c->n_kv_heads) * c->rotary_dim * es + 4.0 * B * kv * es,
               CALL(rope_append(dt, lb.qkv, qkv_dim, c->n_heads, c->n_kv_heads, c->head_dim, c->rotary_dim, B,
                                dec->rows, dec->pos, lb.rope, dec->lens, dec->C_max, dec->kc, dec->vc, dev),
                    "rotary + cache append")));
    TRY(launch(dev, ADADSF_KERNEL_ATTENTION, false, 0,
               (double)B * 2.0 * q * es + 2.0 * B * kv * es * dec->C_max,
               CALL(decode_attention(dt, lb.qkv, qkv_dim, c->n_heads, c->n_kv_heads, c->head_dim, dec->kc,
                                     dec->vc, dec->lens, dec->C_max, B, dec->part_o, dec->part_ml, lb.attn, q,
                                     dev),
                    "decode attention")));
  } else {
    // a6: causal attention among the kept tokens.
    TRY(launch(dev, ADADSF_KERNEL_ATTENTION, tc, 2.0 * B * c->n_heads * c->head_dim * (double)K * (K + 1),
               ((double)M * qkv_dim + (double)M * q) * es,
               CALL(tc ? attention_tc(lb.qkv, qkv_dim, lb.vt, lb.attn, q, B, K, c->n_heads,
                                      c->n_kv_heads, c->head_dim, dev)
                       : attention(dt, lb.qkv, qkv_dim, lb.attn, q, B, K, c->n_heads, c->n_kv_heads,
                                   c->head_dim, dev),
                    "attention")));
  }
  if (sink) {
    // prefill: the kept tokens' keys (rotated) and values, counts and thresholds into the cache
    TRY(launch(dev, ADADSF_KERNEL_KV_CACHE, false, 0, 4.0 * M * kv * es,
               CALL(kv_fill(dt, lb.qkv, qkv_dim, q, kv, B, K, c->head_dim, sink->C_max, sink->kc, sink->vc, dev),
                    "cache fill")));
    TRY(launch(dev, ADADSF_KERNEL_KV_CACHE, false, 0, 8.0 * M,
               CALL(kv_threshold(lb.scores, lb.idx, B, T, K, sink->lens, sink->thr, dev), "cache thresholds")));
  }
  if (neox_tc) {
    // a7 + a8 + a9 as one GEMM with two K sources (parallel residual, Eq. 2):
    // x[row] = x[row] + O W_o^T + act W_down^T + b_o + b_down
    GemmArgs g = linear_args(lb.attn, q, w->w_o, M, d, q);
    g.scratch = lb.split;
    g.scratch_bytes = lb.split ? gemm_split_scratch_bytes() : 0;
    g.A2 = lb.act;
    g.lda2 = F;
    g.Wk2 = w->w_down;
    g.ldwk2 = F;
    g.K2 = F;
    g.epi.bias = w->b_o;
    g.epi.bias2 = w->b_down;
    g.epi.add_rows = x;
    g.epi.ld_add_rows = d;
    g.epi.rows = rows;
    g.epi.out_mapped = true;
    g.epi.out = x;
    g.epi.ld_out = d;
    if (gate) g.epi.gate_scores = lb.scores;   // x[row] + sigmoid(s) delta
    if (lb.cospart) {
      // Eq. 4 partials of (x_in, x_out) per chunk; the residual rows are x_in
      g.epi.cos_out = lb.cospart;
      g.epi.cos_ld = d / 32;
    }
    TRY(launch(dev, ADADSF_KERNEL_GEMM_O_DOWN, true, 2.0 * M * d * ((double)q + F),
               ((double)M * (q + F) + (double)d * (q + F) + 2.0 * Md) * es,
               [&] { return run_linear(dt, g, dev, "output + mlp down projections + residual scatter"); }));
  } else if (neox) {
    // a7: attn_out = O W_o^T + b_o (packed)
    GemmArgs g = linear_args(lb.attn, q, w->w_o, M, d, q);
    g.scratch = lb.split;
    g.scratch_bytes = lb.split ? gemm_split_scratch_bytes() : 0;
    g.epi.bias = w->b_o;
    g.epi.out = lb.ao;
    g.epi.ld_out = d;
    TRY(launch(dev, ADADSF_KERNEL_GEMM_O, tc, 2.0 * M * d * q, ((double)M * q + (double)d * q + Md) * es,
               [&] { return run_linear(dt, g, dev, "output projection"); }));
    // a8: act = GELU(LN2 x W_up^T + b_up)
    GemmArgs u = linear_args(lb.n2, d, w->w_up, M, F, d);
    u.epi.bias = w->b_up;
    u.epi.act = ACT_GELU;
    u.epi.out = lb.act;
    u.epi.ld_out = F;
    TRY(launch(dev, ADADSF_KERNEL_GEMM_UP, tc, 2.0 * M * F * d, (Md + (double)F * d + (double)M * F) * es,
               [&] { return run_linear(dt, u, dev, "mlp up"); }));
    // a8 + a9: x[row] = x[row] + attn_out + act W_down^T + b_down
    GemmArgs dn = linear_args(lb.act, F, w->w_down, M, d, F);
    dn.scratch = lb.split;
    dn.scratch_bytes = lb.split ? gemm_split_scratch_bytes() : 0;
    dn.epi.bias = w->b_down;
    dn.epi.add_packed = lb.ao;
    dn.epi.ld_add_packed = d;
    dn.epi.add_rows = x;
    dn.epi.ld_add_rows = d;
    dn.epi.rows = rows;
    dn.epi.out_mapped = true;
    dn.epi.out = x;
    dn.epi.ld_out = d;
    if (gate) dn.epi.gate_scores = lb.scores;   // x[row] + sigmoid(s) delta
    TRY(launch(dev, ADADSF_KERNEL_GEMM_DOWN, tc, 2.0 * M * d * F,
               ((double)M * F + (double)d * F + 3.0 * Md) * es,
               [&] { return run_linear(dt, dn, dev, "mlp down + residual scatter"); }));
  } else {
    // a7: h = x[row] + O W_o^T (packed)
    GemmArgs g = linear_args(lb.attn, q, w->w_o, M, d, q);
    g.scratch = lb.split;
    g.scratch_bytes = lb.split ? gemm_split_scratch_bytes() : 0;
    g.epi.add_rows = x;
    g.epi.ld_add_rows = d;
    g.epi.rows = rows;
    g.epi.out_mapped = false;
    g.epi.out = lb.ao;
    g.epi.ld_out = d;
    // folded second RMSNorm (bf16), for few rows (a decode step): the O
    // epilogue also leaves each h row's chunk sums of squares and the gate /
    // up epilogue turns them into its rstd, in place of a norm launch. With
    // many rows the two epilogues' extra work costs more than the pass it
    // saves (measured at the Qwen2.5-7B shape), so the pass runs with the
    // folded unit gains.
    const bool fold2 = tc && folded(c) && lb.sq && M <= 128;
    if (fold2) {
      g.epi.sq_out = lb.sq;
      g.epi.sq_ld = d / 32;
    }
    TRY(launch(dev, ADADSF_KERNEL_GEMM_O, tc, 2.0 * M * d * q,
               ((double)M * q + (double)d * q + 2.0 * Md) * es,
               [&] { return run_linear(dt, g, dev, "output projection + residual"); }));
    // a4': RMS2(h) (a pass of its own unless folded)
    if (!fold2)
      TRY(launch(dev, ADADSF_KERNEL_NORM2, false, 0, 2.0 * Md * es,
                 CALL(gather_norm(dt, lb.ao, nullptr, M, d, true, w->ln2_w, nullptr, nullptr, nullptr,
                                  c->norm_eps, lb.n1, nullptr, dev),
                      "post-attention norm")));
    // a8: act = SiLU(h' W_gate^T) * (h' W_up^T)
    GemmArgs u = linear_args(fold2 ? lb.ao : lb.n1, d, w->w_gate, M, F, d);
    u.W2 = w->w_up;
    if (fold2) {
      u.epi.nrm_psum = lb.sq;
      u.epi.nrm_nps = d / 32;
      u.epi.nrm_d = d;
      u.epi.nrm_eps = c->norm_eps;
    }
    u.epi.act = ACT_SWIGLU;
    u.epi.out = lb.act;
    u.epi.ld_out = F;
    TRY(launch(dev, ADADSF_KERNEL_GEMM_UP, tc, 4.0 * M * F * d,
               (Md + 2.0 * F * d + (double)M * F) * es,
               [&] { return run_linear(dt, u, dev, "mlp gate/up"); }));
    // a8 + a9: x[row] = h + act W_down^T
    GemmArgs dn = linear_args(lb.act, F, w->w_down, M, d, F);
    dn.scratch = lb.split;
    dn.scratch_bytes = lb.split ? gemm_split_scratch_bytes() : 0;
    dn.epi.add_packed = lb.ao;
    dn.epi.ld_add_packed = d;
    dn.epi.rows = rows;
    dn.epi.out_mapped = true;
    dn.epi.out = x;
    dn.epi.ld_out = d;
    if (gate) {
      // x[row] + sigmoid(s) (h + mlp - x[row]): the gate scales the whole delta
      dn.epi.gate_scores = lb.scores;
      dn.epi.gate_base = x;
      dn.epi.ld_gate_base = d;
    }
    if (lb.cospart) {
      // Eq. 4 partials of (x_in, x_out) per chunk, x_in read before it is overwritten
      dn.epi.cos_out = lb.cospart;
      dn.epi.cos_ld = d / 32;
      dn.epi.cos_in = x;
      dn.epi.ld_cos_in = d;
    }
    TRY(launch(dev, ADADSF_KERNEL_GEMM_DOWN, tc, 2.0 * M * d * F,
               ((double)M * F + (double)d * F + (gate ? 3.0 : 2.0) * Md) * es,
               [&] { return run_linear(dt, dn, dev, "mlp down + residual scatter"); }));
  }
  return ADADSF_OK;
}

size_t layer_ws_bytes(const adadsf_model_cfg* c, int B, int T, int K) {
  Carver cv;
  cv.take(kErrBytes);
  cv.take(kSyncBytes);   // self-resetting counters (fixed place)
  cv.take(rope_bytes(c, T));
  LayerSlots s;
  carve_layer(c, B, T, K, cv, s);
  return cv.cur;
}

struct ModelSlots {
  size_t x, xin, partials, cospart, rope;
  LayerSlots layer;
  size_t total;
};

void carve_model(const adadsf_model_cfg* c, int B, int T, int Kmax, bool stats, ModelSlots& m) {
  const size_t es = elem_size(c->dtype);
  Carver cv;
  cv.take(kErrBytes);
  cv.take(kSyncBytes);   // self-resetting counters (fixed place)
  m.x = cv.take((size_t)B * T * c->d * es);
  m.xin = stats ? cv.take((size_t)B * T * c->d * es) : 0;
  m.partials = stats ? cv.take((size_t)stats_partials_count((int64_t)B * T) * 3 * 8) : 0;
  // bf16: the Eq. 4 partials of dense layers come from the down epilogue, 16
  // bytes per row and 32-column chunk
  m.cospart = stats && c->dtype == ADADSF_BF16 ? cv.take((size_t)B * T * (c->d / 32) * 16) : 0;
  m.rope = cv.take(rope_bytes(c, T));
  carve_layer(c, B, T, Kmax, cv, m.layer);
  m.total = cv.cur;
}

// ---------------------------------------------------------------- decode cache (see decode.cu)
struct CacheView {
  int32_t* hdr;
  int32_t* lens;   // [L][B]
  float* thr;      // [L][B]
  float2* rope;    // [C_max][rot/2]
  char* kv;        // per layer: K then V, each [B][Hkv][C_max][hd]
  size_t kv_layer_bytes;
  int C_max;
  void* kc(int l) const { return kv + (size_t)l * 2 * kv_layer_bytes; }
  void* vc(int l) const { return kv + (size_t)l * 2 * kv_layer_bytes + kv_layer_bytes; }
};

struct CacheLayout {
  size_t hdr, lens, thr, rope, kv, kv_layer_bytes, total;
};

CacheLayout cache_layout(const adadsf_model_cfg* c, int B, int C_max) {
  CacheLayout cl;
  Carver cv;
  const size_t L = c->n_layers;
  cl.hdr = cv.take(256);
  cl.lens = cv.take(L * B * 4);
  cl.thr = cv.take(L * B * 4);
  cl.rope = cv.take(rope_bytes(c, C_max));
  cl.kv_layer_bytes = align256((size_t)B * c->n_kv_heads * C_max * c->head_dim * elem_size(c->dtype));
  cl.kv = cv.take(2 * L * cl.kv_layer_bytes);
  cl.total = cv.cur;
  return cl;
}

CacheView cache_view(const adadsf_model_cfg* c, int B, int C_max, void* base) {
  const CacheLayout cl = cache_layout(c, B, C_max);
  CacheView v;
  v.hdr = at<int32_t>(base, cl.hdr);
  v.lens = at<int32_t>(base, cl.lens);
  v.thr = at<float>(base, cl.thr);
  v.rope = at<float2>(base, cl.rope);
  v.kv = at<char>(base, cl.kv);
  v.kv_layer_bytes = cl.kv_layer_bytes;
  v.C_max = C_max;
  return v;
}

struct DecodeSlots {
  size_t x, rows, pos, part_o, part_ml;
  LayerSlots layer;
  size_t total;
};

DecodeSlots decode_layout(const adadsf_model_cfg* c, int B) {
  DecodeSlots d;
  Carver cv;
  cv.take(kErrBytes);
  cv.take(kSyncBytes);
  d.x = cv.take((size_t)B * c->d * elem_size(c->dtype));
  d.rows = cv.take((size_t)B * 4);
  d.pos = cv.take((size_t)B * 4);
  // split-attention partials: at most 64 splits per (sequence, query head)
  d.part_o = cv.take((size_t)B * c->n_heads * 64 * c->head_dim * 4);
  d.part_ml = cv.take((size_t)B * c->n_heads * 64 * 8);
  carve_layer(c, B, 1, 1, cv, d.layer);
  d.total = cv.cur;
  return d;
}

adadsf_status model_forward_impl(const adadsf_model_cfg* cfg, const adadsf_model_weights* w,
                                 const int32_t* ids_dev, int B, int T, const int32_t* K_host,
                                 void* hidden_out_dev, double* stats_acc_dev, int32_t* idx_out_dev, void* ws,
                                 size_t ws_bytes, void* stream, const CacheView* cache) {
  TRY(check_cfg(cfg));
  if (!w || !w->layers) return fail(ADADSF_ERR_INVALID_ARG, "model weights or layer array is NULL");
  if (!K_host || cfg->n_layers <= 0) return fail(ADADSF_ERR_INVALID_ARG, "K_host is NULL or n_layers <= 0");
  TRY(check_shape(B, T, 0));
  int kmax = 0;
  for (int l = 0; l < cfg->n_layers; ++l) {
    TRY(check_shape(B, T, K_host[l]));
    if (K_host[l] > 0) TRY(check_layer_weights(cfg, &w->layers[l], K_host[l] < T || gated(cfg)));
    kmax = K_host[l] > kmax ? K_host[l] : kmax;
  }
  NEED_PTR(w->embed, "embed");
  NEED_PTR(w->final_w, "final_w");
  if (cfg->arch == ADADSF_ARCH_NEOX) NEED_PTR(w->final_b, "final_b");
  NEED_PTR(hidden_out_dev, "hidden_out_dev");
  if (cfg->vocab <= 0) return fail(ADADSF_ERR_INVALID_ARG, "vocab <= 0");
  if (B > 0) NEED_PTR(ids_dev, "ids_dev");
  if (stats_acc_dev && (reinterpret_cast<uintptr_t>(stats_acc_dev) & 7u))
    return fail(ADADSF_ERR_INVALID_ARG, "stats_acc_dev misaligned");
  if (idx_out_dev && (reinterpret_cast<uintptr_t>(idx_out_dev) & 3u))
    return fail(ADADSF_ERR_INVALID_ARG, "idx_out_dev misaligned");
  ModelSlots m;
  carve_model(cfg, B, T, kmax, stats_acc_dev != nullptr, m);
  TRY(check_ws(ws, ws_bytes, m.total));
  if (B == 0) return ADADSF_OK;
  Dev dev;
  TRY(device_info(&dev, stream, ws));
  const int dt = cfg->dtype;
  const size_t es = elem_size(dt);
  void* x = at<char>(ws, m.x);
  const double xbytes_d = (double)B * T * cfg->d * es;
  TRY(launch(dev, ADADSF_KERNEL_EMBED, false, 0, 2.0 * xbytes_d + 4.0 * B * T,
             CALL(embed(dt, ids_dev, (int64_t)B * T, w->embed, cfg->vocab, cfg->d, x, dev), "embedding")));
  // the rotary table: T rows in the workspace, or every cache position
  float2* rope_tab = cache ? cache->rope : at<float2>(ws, m.rope);
  const int rope_rows = cache ? cache->C_max : T;
  if (cfg->rotary_dim > 0)
    TRY(launch(dev, ADADSF_KERNEL_ROPE_TABLE, false, 0, rope_bytes(cfg, rope_rows),
               CALL(rope_table(rope_tab, rope_rows, cfg->rotary_dim, cfg->rope_theta, dev), "rotary table")));
  if (cache)
    TRY(launch(dev, ADADSF_KERNEL_KV_CACHE, false, 0, 16.0,
               CALL(cache_header(cache->hdr, T, cache->C_max, cfg->n_layers, B, dev), "cache header")));
  LayerBufs lb;
  lb.scores = at<float>(ws, m.layer.scores);
  lb.rows = at<int32_t>(ws, m.layer.rows);
  lb.rope = rope_tab;
  lb.n1 = at<char>(ws, m.layer.n1);
  lb.n2 = at<char>(ws, m.layer.n2);
  lb.qkv = at<char>(ws, m.layer.qkv);
  lb.vt = at<char>(ws, m.layer.vt);
  lb.attn = at<char>(ws, m.layer.attn);
  lb.ao = at<char>(ws, m.layer.ao);
  lb.act = at<char>(ws, m.layer.act);
  lb.split = m.layer.split ? at<float>(ws, m.layer.split) : nullptr;
  lb.sync = at<int>(ws, kErrBytes);
  lb.rpart = m.layer.rsel ? at<float>(ws, m.layer.rsel) : nullptr;
  lb.sq = m.layer.sq ? at<float>(ws, m.layer.sq) : nullptr;
  lb.tsq = m.layer.tsq ? at<float>(ws, m.layer.tsq) : nullptr;
  const size_t xbytes = (size_t)B * T * cfg->d * es;
  int64_t idx_off = 0;
  for (int l = 0; l < cfg->n_layers; ++l) {
    const int K = K_host[l];
    lb.idx = idx_out_dev ? idx_out_dev + idx_off : at<int32_t>(ws, m.layer.idx);
    // Eq. 4 of a dense bf16 layer: partials from its down-projection epilogue
    // (x_in and x_out are both at hand there); otherwise a copy of the input
    // and a statistics pass
    const bool fused_stats = stats_acc_dev && m.cospart && K == T;
    lb.cospart = fused_stats ? at<float4>(ws, m.cospart) : nullptr;
    if (stats_acc_dev && !fused_stats)
      TRY(launch(dev, ADADSF_KERNEL_COPY, false, 0, 2.0 * xbytes_d,
                 CALL(cudaMemcpyAsync(at<char>(ws, m.xin), x, xbytes, cudaMemcpyDeviceToDevice, dev.stream),
                      "copy of the layer input")));
    CacheSink sink;
    if (cache) {
      sink.kc = cache->kc(l);
      sink.vc = cache->vc(l);
      sink.lens = cache->lens + (int64_t)l * B;
      sink.thr = cache->thr + (int64_t)l * B;
      sink.C_max = cache->C_max;
    }
    TRY(layer_impl(cfg, &w->layers[l], x, B, T, K, lb, idx_out_dev != nullptr, dev, cache ? &sink : nullptr));
    if (fused_stats)
      TRY(launch(dev, ADADSF_KERNEL_STATS, false, 0, 16.0 * B * T * (cfg->d / 32),
                 CALL(cos_stats_chunks(at<float4>(ws, m.cospart), (int64_t)B * T, cfg->d / 32, ADADSF_STATS_TOKEN,
                                       at<double>(ws, m.partials), stats_acc_dev + 2 * l, dev),
                      "similarity statistics")));
    else if (stats_acc_dev)
      TRY(launch(dev, ADADSF_KERNEL_STATS, false, 0, 2.0 * xbytes_d,
                 CALL(cos_stats(dt, at<char>(ws, m.xin), x, (int64_t)B * T, cfg->d, ADADSF_STATS_TOKEN,
                                at<double>(ws, m.partials), stats_acc_dev + 2 * l, dev),
                      "similarity statistics")));
    idx_off += (int64_t)B * K;
  }
  TRY(launch(dev, ADADSF_KERNEL_FINAL_NORM, false, 0, 2.0 * xbytes_d,
             CALL(gather_norm(dt, x, nullptr, (int64_t)B * T, cfg->d, cfg->arch == ADADSF_ARCH_QWEN,
                              w->final_w, w->final_b, nullptr, nullptr, cfg->norm_eps, hidden_out_dev,
                              nullptr, dev),
                  "final norm")));
  return ADADSF_OK;
}

}  // namespace

// ======================================================================== ABI
extern "C" {

const char* adadsf_last_error(void) { return g_last_error.c_str(); }

size_t adadsf_layer_workspace_size(const adadsf_model_cfg* cfg, int B, int T, int K) {
  if (check_cfg(cfg) != ADADSF_OK || check_shape(B, T, K) != ADADSF_OK) return 0;
  return layer_ws_bytes(cfg, B, T, K);
}

size_t adadsf_model_workspace_size(const adadsf_model_cfg* cfg, int B, int T, const int32_t* K_host,
                                   int with_stats) {
  if (check_cfg(cfg) != ADADSF_OK) return 0;
  if (!K_host || cfg->n_layers <= 0) {
    fail(ADADSF_ERR_INVALID_ARG, "K_host is NULL or n_layers <= 0");
    return 0;
  }
  int kmax = 0;
  for (int l = 0; l < cfg->n_layers; ++l) {
    if (check_shape(B, T, K_host[l]) != ADADSF_OK) return 0;
    kmax = K_host[l] > kmax ? K_host[l] : kmax;
  }
  ModelSlots m;
  carve_model(cfg, B, T, kmax, with_stats != 0, m);
  return m.total;
}

size_t adadsf_stats_workspace_size(int64_t n_rows) {
  if (n_rows < 0) return 0;
  return kErrBytes + align256((size_t)stats_partials_count(n_rows) * 3 * 8);
}

adadsf_status adadsf_layer_stats(const void* x_in_dev, const void* x_out_dev, int64_t n_rows, int d,
                                 int dtype, int mode, double* acc_dev, void* ws, size_t ws_bytes,
                                 void* stream) {
  if (dtype != ADADSF_F32 && dtype != ADADSF_BF16)
    return fail(ADADSF_ERR_INVALID_ARG, "dtype %d unknown", dtype);
  if (mode != ADADSF_STATS_TOKEN && mode != ADADSF_STATS_FLAT)
    return fail(ADADSF_ERR_INVALID_ARG, "mode %d unknown", mode);
  if (n_rows < 0 || d <= 0 || d % (dtype == ADADSF_BF16 ? 8 : 4) != 0)
    return fail(ADADSF_ERR_INVALID_ARG, "need n_rows >= 0 and d a positive multiple of 16 bytes");
  if (!acc_dev || (reinterpret_cast<uintptr_t>(acc_dev) & 7u))
    return fail(ADADSF_ERR_INVALID_ARG, "acc_dev is NULL or not 8-byte aligned");
  TRY(check_ws(ws, ws_bytes, adadsf_stats_workspace_size(n_rows)));
  if (n_rows == 0) return ADADSF_OK;
  NEED_PTR(x_in_dev, "x_in_dev");
  NEED_PTR(x_out_dev, "x_out_dev");
  Dev dev;
  TRY(device_info(&dev, stream, ws));
  return launch(dev, ADADSF_KERNEL_STATS, false, 0, 2.0 * n_rows * d * elem_size(dtype),
                CALL(cos_stats(dtype, x_in_dev, x_out_dev, n_rows, d, mode, at<double>(ws, kErrBytes),
                               acc_dev, dev),
                     "similarity statistics"));
}

adadsf_status adadsf_layer_stats_noalloc(const void* x_in_dev, const void* x_out_dev,
                                         int64_t n_rows, int d, int dtype, int mode,
                                         double* acc_dev, void* stream) {
  if (dtype != ADADSF_F32 && dtype != ADADSF_BF16)
    return fail(ADADSF_ERR_INVALID_ARG, "dtype %d unknown", dtype);
  if (mode != ADADSF_STATS_TOKEN && mode != ADADSF_STATS_FLAT)
    return fail(ADADSF_ERR_INVALID_ARG, "mode %d unknown", mode);
  if (n_rows < 0 || d <= 0 || d % (dtype == ADADSF_BF16 ? 8 : 4) != 0)
    return fail(ADADSF_ERR_INVALID_ARG, "need n_rows >= 0 and d a positive multiple of 16 bytes");
  if (n_rows > (int64_t)INT32_MAX)
    return fail(ADADSF_ERR_UNSUPPORTED,
                "workspace-free statistics take n_rows <= %d (got n_rows=%lld)", INT32_MAX,
                (long long)n_rows);
  if (stats_partials_count(n_rows) > stats_static_capacity())
    return fail(ADADSF_ERR_UNSUPPORTED, "needs %d partial-sum slots, the fixed array holds %d",
                stats_partials_count(n_rows), stats_static_capacity());
  if (!acc_dev || (reinterpret_cast<uintptr_t>(acc_dev) & 7u))
    return fail(ADADSF_ERR_INVALID_ARG, "acc_dev is NULL or not 8-byte aligned");
  if (n_rows == 0) return ADADSF_OK;
  NEED_PTR(x_in_dev, "x_in_dev");
  NEED_PTR(x_out_dev, "x_out_dev");
  Dev dev;
  TRY(device_info(&dev, stream, nullptr));
  CUDA_TRY(cos_stats_static(dtype, x_in_dev, x_out_dev, n_rows, d, mode, acc_dev, dev),
           "workspace-free similarity statistics");
  return ADADSF_OK;
}

adadsf_status adadsf_alloc_ratios(const double* s_host, int L, double t, double tau, double beta,
                                  int T, unsigned flags, double* r_out_host, int32_t* K_out_host) {
  if (!s_host || L <= 0) return fail(ADADSF_ERR_INVALID_ARG, "s_host is NULL or L <= 0");
  if (!(t >= 0.0 && t <= 1.0)) return fail(ADADSF_ERR_INVALID_ARG, "t=%g outside [0,1]", t);
  if (!(tau > 0.0) || !(beta > 0.0)) return fail(ADADSF_ERR_INVALID_ARG, "tau and beta must be > 0");
  if (T < 0) return fail(ADADSF_ERR_INVALID_ARG, "T < 0");
  for (int i = 0; i < L; ++i)
    if (!isfinite(s_host[i])) return fail(ADADSF_ERR_INVALID_ARG, "s[%d] is not finite", i);
  // Eq. 5: temperature-normalised weights
  double smax = s_host[0];
  for (int i = 1; i < L; ++i) smax = s_host[i] > smax ? s_host[i] : smax;
  std::vector<double> w(L), rp(L), r(L);
  double wsum = 0.0;
  for (int i = 0; i < L; ++i) {
    w[i] = exp((s_host[i] - smax) / tau);
    wsum += w[i];
  }
  double wmean = 0.0;
  for (int i = 0; i < L; ++i) {
    w[i] /= wsum;
    wmean += w[i];
  }
  wmean /= L;
  // Eqs. 6-7: deviation scaling, sigmoid into (0.05, 0.95)
  double rpsum = 0.0;
  for (int i = 0; i < L; ++i) {
    const double z = beta * (wmean - w[i]);
    rp[i] = 0.05 + 0.9 / (1.0 + exp(-z));
    rpsum += rp[i];
  }
  // Eq. 8: global budget t L
  for (int i = 0; i < L; ++i) r[i] = t * L / rpsum * rp[i];
  if (!(flags & ADADSF_ALLOC_RAW)) {
    if (t >= 1.0) {
      for (int i = 0; i < L; ++i) r[i] = 1.0;
    } else {
      // Clamp to 1, spread the remaining budget over the unclamped layers in
      // proportion to r', until nothing exceeds 1.
      std::vector<char> fixed(L, 0);
      for (;;) {
        bool any = false;
        for (int i = 0; i < L; ++i)
          if (!fixed[i] && r[i] > 1.0) { fixed[i] = 1; any = true; }
        if (!any) break;
        int nfixed = 0;
        double free_rp = 0.0;
        for (int i = 0; i < L; ++i) {
          if (fixed[i]) ++nfixed; else free_rp += rp[i];
        }
        const double budget = t * L - nfixed;
        for (int i = 0; i < L; ++i) r[i] = fixed[i] ? 1.0 : budget / free_rp * rp[i];
      }
    }
  }
  for (int i = 0; i < L; ++i) {
    if (r_out_host) r_out_host[i] = r[i];
    if (K_out_host) {
      double k = (flags & ADADSF_ALLOC_ROUND) ? floor(r[i] * T + 0.5) : floor(r[i] * T + 1e-9);
      if (k < 0) k = 0;
      if (k > T) k = T;
      K_out_host[i] = (int32_t)k;
    }
  }
  return ADADSF_OK;
}

adadsf_status adadsf_similarity(const double* acc_host, int L, int mode, double* s_out_host) {
  if (!acc_host || !s_out_host || L <= 0)
    return fail(ADADSF_ERR_INVALID_ARG, "acc_host / s_out_host is NULL or L <= 0");
  if (mode != ADADSF_STATS_TOKEN && mode != ADADSF_STATS_FLAT)
    return fail(ADADSF_ERR_INVALID_ARG, "mode %d unknown", mode);
  for (int l = 0; l < L; ++l) {
    if (mode == ADADSF_STATS_TOKEN) {
      // Eq. 4, token mode: mean of the per-token cosines
      const double sum = acc_host[2 * l], n = acc_host[2 * l + 1];
      if (!(n > 0.0)) return fail(ADADSF_ERR_INVALID_ARG, "layer %d: token count %g is not positive", l, n);
      s_out_host[l] = sum / n;
    } else {
      // Eq. 4, flat mode: cosine of the flattened tensors, zero norms guarded
      const double dot = acc_host[3 * l], na = sqrt(acc_host[3 * l + 1]), nb = sqrt(acc_host[3 * l + 2]);
      s_out_host[l] = dot / ((na > 1e-8 ? na : 1e-8) * (nb > 1e-8 ? nb : 1e-8));
    }
    if (!isfinite(s_out_host[l])) return fail(ADADSF_ERR_INVALID_ARG, "layer %d: similarity is not finite", l);
  }
  return ADADSF_OK;
}

adadsf_status adadsf_fold_norms(const adadsf_model_cfg* cfg, const adadsf_layer_weights* w, void* stream) {
  TRY(check_cfg(cfg));
  TRY(check_layer_weights(cfg, w, false));
  const bool neox = cfg->arch == ADADSF_ARCH_NEOX;
  if (neox) {
    NEED_PTR(w->b_qkv, "b_qkv");
    NEED_PTR(w->b_up, "b_up");
  }
  Dev dev;
  TRY(device_info(&dev, stream, nullptr));
  const int qkv = (cfg->n_heads + 2 * cfg->n_kv_heads) * cfg->head_dim;
  auto mut = [](const void* p) { return const_cast<void*>(p); };
  CUDA_TRY(fold_layer_norms(cfg->dtype, neox, cfg->d, qkv, cfg->ffn, mut(w->w_qkv), mut(w->b_qkv), mut(w->w_up),
                            mut(w->b_up), mut(w->w_gate), mut(w->ln1_w), mut(w->ln1_b), mut(w->ln2_w),
                            mut(w->ln2_b), dev),
           "norm folding");
  return ADADSF_OK;
}

size_t adadsf_align_workspace_size(int64_t n_rows, int n_classes) {
  if (n_rows < 0 || n_classes < 0) return 0;
  return kErrBytes + kSyncBytes + align256((size_t)train_row_blocks(n_rows) * 8) +
         2 * align256((size_t)n_rows * n_classes * 4);
}

adadsf_status adadsf_align_hidden(const void* hs_dev, const void* hd_dev, int64_t n_rows, int d, int dtype,
                                  double* acc_dev, float* grad_dev, void* ws, size_t ws_bytes, void* stream) {
  if (dtype != ADADSF_F32 && dtype != ADADSF_BF16) return fail(ADADSF_ERR_INVALID_ARG, "dtype %d unknown", dtype);
  if (n_rows < 0 || d <= 0) return fail(ADADSF_ERR_INVALID_ARG, "need n_rows >= 0 and d > 0");
  if (!acc_dev || (reinterpret_cast<uintptr_t>(acc_dev) & 7u))
    return fail(ADADSF_ERR_INVALID_ARG, "acc_dev is NULL or not 8-byte aligned");
  TRY(check_ws(ws, ws_bytes, adadsf_align_workspace_size(n_rows, 0)));
  if (n_rows == 0) return ADADSF_OK;
  NEED_PTR(hs_dev, "hs_dev");
  NEED_PTR(hd_dev, "hd_dev");
  if (grad_dev && (reinterpret_cast<uintptr_t>(grad_dev) & 3u))
    return fail(ADADSF_ERR_INVALID_ARG, "grad_dev misaligned");
  Dev dev;
  TRY(device_info(&dev, stream, ws));
  return launch(dev, ADADSF_KERNEL_ALIGN, false, 0, (2.0 + (grad_dev ? 2.0 : 0.0)) * n_rows * d * elem_size(dtype),
                CALL(align_hidden(dtype, hs_dev, hd_dev, n_rows, d, grad_dev, at<double>(ws, kErrBytes + kSyncBytes),
                                  acc_dev, dev),
                     "hidden-state alignment"));
}

adadsf_status adadsf_align_output(const void* hs_dev, const void* hd_dev, const void* w_head_dev, int64_t n_rows,
                                  int d, int n_classes, int dtype, double* acc_dev, void* ws, size_t ws_bytes,
                                  void* stream) {
  if (dtype != ADADSF_F32 && dtype != ADADSF_BF16) return fail(ADADSF_ERR_INVALID_ARG, "dtype %d unknown", dtype);
  if (n_rows < 0 || d <= 0 || n_classes <= 0) return fail(ADADSF_ERR_INVALID_ARG, "need n_rows >= 0, d, n_classes > 0");
  if (dtype == ADADSF_BF16 ? (d % 64 || n_classes % 64) : (d % 4 || n_classes % 4))
    return fail(ADADSF_ERR_UNSUPPORTED, "d and n_classes must be multiples of %d", dtype == ADADSF_BF16 ? 64 : 4);
  if (n_rows > (int64_t)INT32_MAX) return fail(ADADSF_ERR_UNSUPPORTED, "n_rows too large");
  if (!acc_dev || (reinterpret_cast<uintptr_t>(acc_dev) & 7u))
    return fail(ADADSF_ERR_INVALID_ARG, "acc_dev is NULL or not 8-byte aligned");
  TRY(check_ws(ws, ws_bytes, adadsf_align_workspace_size(n_rows, n_classes)));
  if (n_rows == 0) return ADADSF_OK;
  NEED_PTR(hs_dev, "hs_dev");
  NEED_PTR(hd_dev, "hd_dev");
  NEED_PTR(w_head_dev, "w_head_dev");
  Dev dev;
  TRY(device_info(&dev, stream, ws));
  Carver cv;
  cv.take(kErrBytes);
  cv.take(kSyncBytes);
  const size_t part = cv.take((size_t)train_row_blocks(n_rows) * 8);
  const size_t ls = cv.take((size_t)n_rows * n_classes * 4);
  const size_t ld = cv.take((size_t)n_rows * n_classes * 4);
  // logits h W_head^T of both models, fp32
  for (int k = 0; k < 2; ++k) {
    GemmArgs g = linear_args(k == 0 ? hs_dev : hd_dev, d, w_head_dev, n_rows, n_classes, d);
    float* lg = at<float>(ws, k == 0 ? ls : ld);
    if (dtype == ADADSF_BF16) {
      g.epi.out_f32 = lg;
      g.epi.ld_out = n_classes;
    } else {
      g.epi.out = lg;
      g.epi.ld_out = n_classes;
    }
    TRY(launch(dev, ADADSF_KERNEL_LINEAR, dtype == ADADSF_BF16, 2.0 * n_rows * n_classes * d,
               ((double)n_rows * d + (double)n_classes * d) * elem_size(dtype) + 4.0 * n_rows * n_classes,
               [&] { return run_linear(dtype, g, dev, "head logits"); }));
  }
  return launch(dev, ADADSF_KERNEL_ALIGN, false, 0, 8.0 * n_rows * n_classes,
                CALL(kl_rows(at<float>(ws, ls), at<float>(ws, ld), n_rows, n_classes, at<double>(ws, part), acc_dev,
                             dev),
                     "output alignment"));
}

size_t adadsf_router_backward_workspace_size(const adadsf_model_cfg* cfg, int64_t n_kept) {
  if (check_cfg(cfg) != ADADSF_OK || n_kept < 0) return 0;
  const size_t h = cfg->router_hidden;
  return kErrBytes + align256((size_t)n_kept * h * 4) * 2 + align256((size_t)n_kept * 4);
}

adadsf_status adadsf_router_backward(const adadsf_model_cfg* cfg, const adadsf_layer_weights* w, const void* x_dev,
                                     const void* y_plain_dev, const int32_t* rows_dev, int64_t n_kept,
                                     const float* grad_y_dev, float* grad_out_dev, void* ws, size_t ws_bytes,
                                     void* stream) {
  TRY(check_cfg(cfg));
  if (!w) return fail(ADADSF_ERR_INVALID_ARG, "weights are NULL");
  NEED_PTR(w->router_w1, "router_w1");
  NEED_PTR(w->router_b1, "router_b1");
  NEED_PTR(w->router_w2, "router_w2");
  if (!w->router_b2) return fail(ADADSF_ERR_INVALID_ARG, "router_b2 is NULL");
  if (cfg->router_hidden > 64) return fail(ADADSF_ERR_UNSUPPORTED, "router_hidden > 64");
  if (n_kept < 0) return fail(ADADSF_ERR_INVALID_ARG, "n_kept < 0");
  NEED_PTR(grad_out_dev, "grad_out_dev");
  TRY(check_ws(ws, ws_bytes, adadsf_router_backward_workspace_size(cfg, n_kept)));
  if (n_kept > 0) {
    NEED_PTR(x_dev, "x_dev");
    NEED_PTR(y_plain_dev, "y_plain_dev");
    if (!rows_dev) return fail(ADADSF_ERR_INVALID_ARG, "rows_dev is NULL");
    if (!grad_y_dev) return fail(ADADSF_ERR_INVALID_ARG, "grad_y_dev is NULL");
  }
  Dev dev;
  TRY(device_info(&dev, stream, ws));
  const int h = cfg->router_hidden, d = cfg->d;
  Carver cv;
  cv.take(kErrBytes);
  float* du = at<float>(ws, cv.take((size_t)n_kept * h * 4));
  float* su = at<float>(ws, cv.take((size_t)n_kept * h * 4));
  float* ds = at<float>(ws, cv.take((size_t)n_kept * 4));
  return launch(dev, ADADSF_KERNEL_ALIGN, false, 4.0 * n_kept * h * d,
                (double)n_kept * d * (2.0 * elem_size(cfg->dtype) + 4.0),
                CALL(router_backward(cfg->dtype, x_dev, y_plain_dev, rows_dev, n_kept, d, h, w->router_w1,
                                     w->router_b1, w->router_w2, w->router_b2, grad_y_dev, du, su, ds, grad_out_dev,
                                     dev),
                     "router backward"));
}

adadsf_status adadsf_normalized_flops(const adadsf_model_cfg* cfg, int T, const int32_t* K_host,
                                      double* out_host) {
  TRY(check_cfg(cfg));
  if (!K_host || !out_host || cfg->n_layers <= 0)
    return fail(ADADSF_ERR_INVALID_ARG, "K_host / out_host is NULL or n_layers <= 0");
  if (T <= 0) return fail(ADADSF_ERR_INVALID_ARG, "T=%d must be positive", T);
  const double d = cfg->d, hd = cfg->head_dim, F = cfg->ffn;
  const double q = (double)cfg->n_heads * hd, kv = (double)cfg->n_kv_heads * hd;
  const double n_mlp = cfg->arch == ADADSF_ARCH_QWEN ? 3.0 : 2.0;
  // one layer on K tokens of a sequence: projections + causal attention
  auto block = [&](double K) {
    return 2.0 * K * ((q + 2.0 * kv) * d + d * q + n_mlp * d * F) + 2.0 * q * K * (K + 1.0);
  };
  const double router = 2.0 * T * cfg->router_hidden * (d + 1.0);
  double num = 0.0;
  for (int l = 0; l < cfg->n_layers; ++l) {
    const int K = K_host[l];
    if (K < 0 || K > T) return fail(ADADSF_ERR_INVALID_ARG, "K[%d]=%d outside [0, T=%d]", l, K, T);
    num += (K < T ? router : 0.0) + block(K);
  }
  *out_host = num / (cfg->n_layers * block(T));
  return ADADSF_OK;
}

adadsf_status adadsf_router_scores(const adadsf_model_cfg* cfg, const adadsf_layer_weights* w,
                                   const void* x_dev, int64_t n_rows, float* scores_dev, void* ws,
                                   size_t ws_bytes, void* stream) {
  TRY(check_cfg(cfg));
  if (!w) return fail(ADADSF_ERR_INVALID_ARG, "weights are NULL");
  if (n_rows < 0 || n_rows > ((int64_t)1 << 30)) return fail(ADADSF_ERR_INVALID_ARG, "n_rows out of range");
  TRY(check_ws(ws, ws_bytes, kErrBytes));
  if (n_rows == 0) return ADADSF_OK;
  NEED_PTR(x_dev, "x_dev");
  NEED_PTR(scores_dev, "scores_dev");
  NEED_PTR(w->router_w1, "router_w1");
  NEED_PTR(w->router_b1, "router_b1");
  NEED_PTR(w->router_w2, "router_w2");
  if (!w->router_b2) return fail(ADADSF_ERR_INVALID_ARG, "router_b2 is NULL");
  Dev dev;
  TRY(device_info(&dev, stream, ws));
  if (cfg->dtype == ADADSF_BF16) {
    // with room for them: counters (synchronisation area) and partial tiles
    // for 128-token tiles split along d
    const bool split = ws_bytes >= kErrBytes + kSyncBytes + router_partial_bytes();
    CUDA_TRY(router_tc(x_dev, n_rows, cfg->d, w->router_w1, w->router_b1, w->router_w2, w->router_b2,
                       scores_dev, nullptr, split ? at<int>(ws, kErrBytes) : nullptr,
                       split ? at<float>(ws, kErrBytes + kSyncBytes) : nullptr, dev),
             "router");
    return ADADSF_OK;
  }
  CUDA_TRY(router_f32(static_cast<const float*>(x_dev), n_rows, cfg->d, cfg->router_hidden,
                      static_cast<const float*>(w->router_w1), static_cast<const float*>(w->router_b1),
                      static_cast<const float*>(w->router_w2), static_cast<const float*>(w->router_b2),
                      scores_dev, dev),
           "router");
  return ADADSF_OK;
}

adadsf_status adadsf_topk_select(const float* scores_dev, int B, int T, int K, int32_t* idx_dev,
                                 int32_t* rows_dev, void* stream) {
  TRY(check_shape(B, T, K));
  if (B == 0 || K == 0) return ADADSF_OK;
  NEED_PTR(scores_dev, "scores_dev");
  if (!idx_dev || (reinterpret_cast<uintptr_t>(idx_dev) & 3u))
    return fail(ADADSF_ERR_INVALID_ARG, "idx_dev is NULL or misaligned");
  Dev dev;
  TRY(device_info(&dev, stream, nullptr));
  CUDA_TRY(topk(scores_dev, B, T, K, idx_dev, rows_dev, dev), "top-k");
  return ADADSF_OK;
}

size_t adadsf_router_select_workspace_size(const adadsf_model_cfg* cfg, int B, int T) {
  if (check_cfg(cfg) != ADADSF_OK || check_shape(B, T, 0) != ADADSF_OK) return 0;
  return kErrBytes + kSyncBytes + (cfg->dtype == ADADSF_BF16 ? align256(router_partial_bytes()) : 0);
}

adadsf_status adadsf_router_select(const adadsf_model_cfg* cfg, const adadsf_layer_weights* w,
                                   const void* x_dev, int B, int T, int K, float* scores_dev,
                                   int32_t* idx_dev, int32_t* rows_dev, void* ws, size_t ws_bytes,
                                   void* stream) {
  TRY(check_cfg(cfg));
  if (!w) return fail(ADADSF_ERR_INVALID_ARG, "weights are NULL");
  TRY(check_shape(B, T, K));
  if (B == 0) return ADADSF_OK;
  if (K < 1) return fail(ADADSF_ERR_INVALID_ARG, "K must be at least 1");
  TRY(check_ws(ws, ws_bytes, adadsf_router_select_workspace_size(cfg, B, T)));
  NEED_PTR(x_dev, "x_dev");
  NEED_PTR(scores_dev, "scores_dev");
  if (!idx_dev || (reinterpret_cast<uintptr_t>(idx_dev) & 3u))
    return fail(ADADSF_ERR_INVALID_ARG, "idx_dev is NULL or misaligned");
  if (rows_dev && (reinterpret_cast<uintptr_t>(rows_dev) & 3u))
    return fail(ADADSF_ERR_INVALID_ARG, "rows_dev misaligned");
  NEED_PTR(w->router_w1, "router_w1");
  NEED_PTR(w->router_b1, "router_b1");
  NEED_PTR(w->router_w2, "router_w2");
  if (!w->router_b2) return fail(ADADSF_ERR_INVALID_ARG, "router_b2 is NULL");
  Dev dev;
  TRY(device_info(&dev, stream, ws));
  const int64_t BT = (int64_t)B * T;
  if (cfg->dtype == ADADSF_BF16)
    CUDA_TRY(router_tc(x_dev, BT, cfg->d, w->router_w1, w->router_b1, w->router_w2, w->router_b2,
                       scores_dev, nullptr, at<int>(ws, kErrBytes), at<float>(ws, kErrBytes + kSyncBytes), dev),
             "router");
  else
    CUDA_TRY(router_f32(static_cast<const float*>(x_dev), BT, cfg->d, cfg->router_hidden,
                      static_cast<const float*>(w->router_w1), static_cast<const float*>(w->router_b1),
                      static_cast<const float*>(w->router_w2), static_cast<const float*>(w->router_b2),
                      scores_dev, dev),
           "router");
  CUDA_TRY(topk(scores_dev, B, T, K, idx_dev, rows_dev, dev), "top-k");
  return ADADSF_OK;
}

adadsf_status adadsf_linear(const void* x_dev, const void* w_dev, const void* bias_dev, int64_t M,
                            int n_out, int k_in, int dtype, int act, void* out_dev, void* ws,
                            size_t ws_bytes, void* stream) {
  if (dtype != ADADSF_F32 && dtype != ADADSF_BF16)
    return fail(ADADSF_ERR_INVALID_ARG, "dtype %d unknown", dtype);
  if (act != 0 && act != 1) return fail(ADADSF_ERR_INVALID_ARG, "act %d unknown", act);
  const int mult = dtype == ADADSF_BF16 ? 64 : 4;
  if (M < 0 || M > ((int64_t)1 << 30) || n_out <= 0 || k_in <= 0 || n_out % mult || k_in % mult)
    return fail(ADADSF_ERR_UNSUPPORTED, "need M >= 0 and n_out, k_in positive multiples of %d", mult);
  TRY(check_ws(ws, ws_bytes, kErrBytes));
  if (M == 0) return ADADSF_OK;
  NEED_PTR(x_dev, "x_dev");
  NEED_PTR(w_dev, "w_dev");
  NEED_PTR(out_dev, "out_dev");
  if (bias_dev && !aligned16(bias_dev)) return fail(ADADSF_ERR_INVALID_ARG, "bias_dev misaligned");
  Dev dev;
  TRY(device_info(&dev, stream, ws));
  GemmArgs g = linear_args(x_dev, k_in, w_dev, M, n_out, k_in);
  if (dtype == ADADSF_BF16 && ws_bytes > kErrBytes) {   // the rest of ws: split-K scratch
    g.scratch = at<float>(ws, kErrBytes);
    g.scratch_bytes = ws_bytes - kErrBytes;
  }
  g.epi.bias = bias_dev;
  g.epi.act = act == 1 ? ACT_GELU : ACT_NONE;
  g.epi.out = out_dev;
  g.epi.ld_out = n_out;
  const double es = elem_size(dtype);
  return launch(dev, ADADSF_KERNEL_LINEAR, dtype == ADADSF_BF16, 2.0 * M * n_out * k_in,
                ((double)M * k_in + (double)n_out * k_in + (double)M * n_out) * es,
                [&] { return run_linear(dtype, g, dev, "linear"); });
}

size_t adadsf_attention_workspace_size(const adadsf_model_cfg* cfg, int B, int K) {
  if (check_cfg(cfg) != ADADSF_OK || B < 0 || K < 0) return 0;
  const size_t kv = (size_t)cfg->n_kv_heads * cfg->head_dim;
  return kErrBytes + (cfg->dtype == ADADSF_BF16 ? align256((size_t)B * kv * vt_pad(K) * 2) : 0);
}

adadsf_status adadsf_causal_attention(const adadsf_model_cfg* cfg, const void* qkv_dev, int B, int K,
                                      void* out_dev, void* ws, size_t ws_bytes, void* stream) {
  TRY(check_cfg(cfg));
  if (B < 0 || K < 0 || (int64_t)B * K > ((int64_t)1 << 30))
    return fail(ADADSF_ERR_INVALID_ARG, "B and K must be >= 0");
  TRY(check_ws(ws, ws_bytes, adadsf_attention_workspace_size(cfg, B, K)));
  if (B == 0 || K == 0) return ADADSF_OK;
  NEED_PTR(qkv_dev, "qkv_dev");
  NEED_PTR(out_dev, "out_dev");
  Dev dev;
  TRY(device_info(&dev, stream, ws));
  const int q = cfg->n_heads * cfg->head_dim, kv = cfg->n_kv_heads * cfg->head_dim;
  const double flops = 2.0 * B * cfg->n_heads * cfg->head_dim * (double)K * (K + 1);
  const double es = elem_size(cfg->dtype);
  const double bytes = (double)B * K * (q + 2.0 * kv + q) * es;
  if (cfg->dtype == ADADSF_BF16) {
    void* vt = at<char>(ws, kErrBytes);
    TRY(launch(dev, ADADSF_KERNEL_COPY, false, 0, 2.0 * B * K * kv * es,
               CALL(vt_from_qkv(qkv_dev, q + 2 * kv, q + kv, B, K, cfg->n_kv_heads, cfg->head_dim, vt,
                                dev),
                    "value transpose")));
    return launch(dev, ADADSF_KERNEL_ATTENTION, true, flops, bytes,
                  CALL(attention_tc(qkv_dev, q + 2 * kv, vt, out_dev, q, B, K, cfg->n_heads,
                                    cfg->n_kv_heads, cfg->head_dim, dev),
                       "attention"));
  }
  CUDA_TRY(attention(cfg->dtype, qkv_dev, q + 2 * kv, out_dev, q, B, K, cfg->n_heads,
                     cfg->n_kv_heads, cfg->head_dim, dev),
           "attention");
  return ADADSF_OK;
}

adadsf_status adadsf_sparse_layer_forward(const adadsf_model_cfg* cfg, const adadsf_layer_weights* w,
                                          void* x_dev, int B, int T, int K, int32_t* idx_out_dev,
                                          float* scores_out_dev, void* ws, size_t ws_bytes,
                                          void* stream) {
  TRY(check_cfg(cfg));
  TRY(check_shape(B, T, K));
  if (K == 0 || B == 0) return ADADSF_OK;
  TRY(check_layer_weights(cfg, w, K < T || gated(cfg)));
  NEED_PTR(x_dev, "x_dev");
  if (idx_out_dev && (reinterpret_cast<uintptr_t>(idx_out_dev) & 3u))
    return fail(ADADSF_ERR_INVALID_ARG, "idx_out_dev misaligned");
  if (scores_out_dev && (reinterpret_cast<uintptr_t>(scores_out_dev) & 3u))
    return fail(ADADSF_ERR_INVALID_ARG, "scores_out_dev misaligned");
  TRY(check_ws(ws, ws_bytes, layer_ws_bytes(cfg, B, T, K)));
  Dev dev;
  TRY(device_info(&dev, stream, ws));
  Carver cv;
  cv.take(kErrBytes);
  cv.take(kSyncBytes);   // self-resetting counters (fixed place)
  const size_t rope_off = cv.take(rope_bytes(cfg, T));
  LayerSlots s;
  carve_layer(cfg, B, T, K, cv, s);
  LayerBufs lb;
  lb.scores = scores_out_dev ? scores_out_dev : at<float>(ws, s.scores);
  lb.idx = idx_out_dev ? idx_out_dev : at<int32_t>(ws, s.idx);
  lb.rows = at<int32_t>(ws, s.rows);
  lb.rope = at<float2>(ws, rope_off);
  lb.n1 = at<char>(ws, s.n1);
  lb.n2 = at<char>(ws, s.n2);
  lb.qkv = at<char>(ws, s.qkv);
  lb.vt = at<char>(ws, s.vt);
  lb.attn = at<char>(ws, s.attn);
  lb.ao = at<char>(ws, s.ao);
  lb.act = at<char>(ws, s.act);
  lb.split = s.split ? at<float>(ws, s.split) : nullptr;
  lb.sync = at<int>(ws, kErrBytes);
  lb.rpart = s.rsel ? at<float>(ws, s.rsel) : nullptr;
  lb.sq = s.sq ? at<float>(ws, s.sq) : nullptr;
  lb.tsq = s.tsq ? at<float>(ws, s.tsq) : nullptr;
  if (cfg->rotary_dim > 0)
    TRY(launch(dev, ADADSF_KERNEL_ROPE_TABLE, false, 0, rope_bytes(cfg, T),
               CALL(rope_table(at<float2>(ws, rope_off), T, cfg->rotary_dim, cfg->rope_theta, dev),
                    "rotary table")));
  return layer_impl(cfg, w, x_dev, B, T, K, lb, idx_out_dev != nullptr, dev);
}

adadsf_status adadsf_sparse_model_forward(const adadsf_model_cfg* cfg, const adadsf_model_weights* w,
                                          const int32_t* ids_dev, int B, int T, const int32_t* K_host,
                                          void* hidden_out_dev, double* stats_acc_dev,
                                          int32_t* idx_out_dev, void* ws, size_t ws_bytes,
                                          void* stream) {
  return model_forward_impl(cfg, w, ids_dev, B, T, K_host, hidden_out_dev, stats_acc_dev, idx_out_dev, ws,
                            ws_bytes, stream, nullptr);
}

size_t adadsf_kv_cache_size(const adadsf_model_cfg* cfg, int B, int C_max) {
  if (check_cfg(cfg) != ADADSF_OK) return 0;
  if (B <= 0 || C_max <= 0 || C_max > 65536 || cfg->n_layers <= 0) {
    fail(ADADSF_ERR_INVALID_ARG, "need B > 0, 0 < C_max <= 65536 and n_layers > 0");
    return 0;
  }
  return cache_layout(cfg, B, C_max).total;
}

adadsf_status adadsf_prefill(const adadsf_model_cfg* cfg, const adadsf_model_weights* w, const int32_t* ids_dev,
                             int B, int T, const int32_t* K_host, void* hidden_out_dev, int32_t* idx_out_dev,
                             void* cache_dev, size_t cache_bytes, int C_max, void* ws, size_t ws_bytes,
                             void* stream) {
  TRY(check_cfg(cfg));
  if (B <= 0) return fail(ADADSF_ERR_INVALID_ARG, "B=%d must be positive", B);
  if (T <= 0 || T >= C_max)
    return fail(ADADSF_ERR_INVALID_ARG, "need 0 < T < C_max (T=%d, C_max=%d): room for generated tokens", T, C_max);
  const size_t need = adadsf_kv_cache_size(cfg, B, C_max);
  if (need == 0) return ADADSF_ERR_INVALID_ARG;
  if (!cache_dev || (reinterpret_cast<uintptr_t>(cache_dev) & 255u))
    return fail(ADADSF_ERR_INVALID_ARG, "cache_dev is NULL or not 256-byte aligned");
  if (cache_bytes < need)
    return fail(ADADSF_ERR_WORKSPACE_TOO_SMALL, "cache has %zu bytes, needs %zu", cache_bytes, need);
  const CacheView cv = cache_view(cfg, B, C_max, cache_dev);
  return model_forward_impl(cfg, w, ids_dev, B, T, K_host, hidden_out_dev, nullptr, idx_out_dev, ws, ws_bytes,
                            stream, &cv);
}

size_t adadsf_decode_workspace_size(const adadsf_model_cfg* cfg, int B, int C_max) {
  if (check_cfg(cfg) != ADADSF_OK) return 0;
  if (B <= 0 || C_max <= 0) {
    fail(ADADSF_ERR_INVALID_ARG, "need B > 0 and C_max > 0");
    return 0;
  }
  return decode_layout(cfg, B).total;
}

adadsf_status adadsf_decode_step(const adadsf_model_cfg* cfg, const adadsf_model_weights* w, const int32_t* ids_dev,
                                 int B, void* hidden_out_dev, int32_t* kept_out_dev, void* cache_dev,
                                 size_t cache_bytes, int C_max, void* ws, size_t ws_bytes, void* stream) {
  TRY(check_cfg(cfg));
  if (cfg->n_heads / cfg->n_kv_heads > 16)
    return fail(ADADSF_ERR_UNSUPPORTED, "decode takes at most 16 query heads per key/value head, not %d",
                cfg->n_heads / cfg->n_kv_heads);
  if (!w || !w->layers) return fail(ADADSF_ERR_INVALID_ARG, "model weights or layer array is NULL");
  if (B <= 0) return fail(ADADSF_ERR_INVALID_ARG, "B=%d must be positive", B);
  for (int l = 0; l < cfg->n_layers; ++l) TRY(check_layer_weights(cfg, &w->layers[l], true));
  NEED_PTR(w->embed, "embed");
  NEED_PTR(w->final_w, "final_w");
  if (cfg->arch == ADADSF_ARCH_NEOX) NEED_PTR(w->final_b, "final_b");
  NEED_PTR(ids_dev, "ids_dev");
  NEED_PTR(hidden_out_dev, "hidden_out_dev");
  if (kept_out_dev && (reinterpret_cast<uintptr_t>(kept_out_dev) & 3u))
    return fail(ADADSF_ERR_INVALID_ARG, "kept_out_dev misaligned");
  const size_t need = adadsf_kv_cache_size(cfg, B, C_max);
  if (need == 0) return ADADSF_ERR_INVALID_ARG;
  if (!cache_dev || (reinterpret_cast<uintptr_t>(cache_dev) & 255u))
    return fail(ADADSF_ERR_INVALID_ARG, "cache_dev is NULL or not 256-byte aligned");
  if (cache_bytes < need)
    return fail(ADADSF_ERR_WORKSPACE_TOO_SMALL, "cache has %zu bytes, needs %zu", cache_bytes, need);
  const DecodeSlots ds = decode_layout(cfg, B);
  TRY(check_ws(ws, ws_bytes, ds.total));
  Dev dev;
  TRY(device_info(&dev, stream, ws));
  const CacheView cv = cache_view(cfg, B, C_max, cache_dev);
  const int dt = cfg->dtype;
  const double es = elem_size(dt);
  void* x = at<char>(ws, ds.x);
  TRY(launch(dev, ADADSF_KERNEL_EMBED, false, 0, 2.0 * B * cfg->d * es + 4.0 * B,
             CALL(embed(dt, ids_dev, B, w->embed, cfg->vocab, cfg->d, x, dev), "embedding")));
  LayerBufs lb;
  lb.scores = at<float>(ws, ds.layer.scores);
  lb.idx = at<int32_t>(ws, ds.layer.idx);
  lb.rows = at<int32_t>(ws, ds.layer.rows);
  lb.rope = cv.rope;
  lb.n1 = at<char>(ws, ds.layer.n1);
  lb.n2 = at<char>(ws, ds.layer.n2);
  lb.qkv = at<char>(ws, ds.layer.qkv);
  lb.vt = at<char>(ws, ds.layer.vt);
  lb.attn = at<char>(ws, ds.layer.attn);
  lb.ao = at<char>(ws, ds.layer.ao);
  lb.act = at<char>(ws, ds.layer.act);
  lb.split = ds.layer.split ? at<float>(ws, ds.layer.split) : nullptr;
  lb.sync = at<int>(ws, kErrBytes);
  lb.rpart = ds.layer.rsel ? at<float>(ws, ds.layer.rsel) : nullptr;
  lb.sq = ds.layer.sq ? at<float>(ws, ds.layer.sq) : nullptr;
  lb.tsq = ds.layer.tsq ? at<float>(ws, ds.layer.tsq) : nullptr;
  cudaStream_t side = nullptr;
  cudaEvent_t ev_fork = nullptr, ev_join = nullptr;
  const bool has_side = decode_side_stream(dev.stream, &side, &ev_fork, &ev_join);
  for (int l = 0; l < cfg->n_layers; ++l) {
    DecodeCtx dc;
    dc.thr = cv.thr + (int64_t)l * B;
    dc.hdr = cv.hdr;
    dc.lens = cv.lens + (int64_t)l * B;
    dc.kc = cv.kc(l);
    dc.vc = cv.vc(l);
    dc.C_max = C_max;
    dc.rows = at<int32_t>(ws, ds.rows);
    dc.pos = at<int32_t>(ws, ds.pos);
    dc.part_o = at<float>(ws, ds.part_o);
    dc.part_ml = at<float2>(ws, ds.part_ml);
    dc.kept_out = kept_out_dev ? kept_out_dev + (int64_t)l * B : nullptr;
    if (has_side) {
      dc.side = side;
      dc.fork = ev_fork;
      dc.join = ev_join;
    }
    TRY(layer_impl(cfg, &w->layers[l], x, B, 1, 1, lb, false, dev, nullptr, &dc));
  }
  TRY(launch(dev, ADADSF_KERNEL_FINAL_NORM, false, 0, 2.0 * B * cfg->d * es,
             CALL(gather_norm(dt, x, nullptr, B, cfg->d, cfg->arch == ADADSF_ARCH_QWEN, w->final_w, w->final_b,
                              nullptr, nullptr, cfg->norm_eps, hidden_out_dev, nullptr, dev),
                  "final norm")));
  TRY(launch(dev, ADADSF_KERNEL_KV_CACHE, false, 0, 8.0, CALL(decode_advance(cv.hdr, dev), "advance position")));
  return ADADSF_OK;
}

adadsf_status adadsf_sync_check(void* ws, size_t ws_bytes, void* stream) {
  TRY(check_ws(ws, ws_bytes, kErrBytes));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int h = 0;
  CUDA_TRY(cudaMemcpyAsync(&h, ws, sizeof(int), cudaMemcpyDeviceToHost, s), "read error word");
  CUDA_TRY(cudaStreamSynchronize(s), "stream synchronise");
  if (h != 0) {
    CUDA_TRY(cudaMemsetAsync(ws, 0, sizeof(int), s), "clear error word");
    // A kernel that gave up may have left arrival counters of the
    // synchronisation area part-way (other CTAs of the same tile had already
    // counted): zero them so the workspace is valid for the next call.
    if ((h & DEVERR_TIMEOUT) && ws_bytes >= kErrBytes + kSyncBytes)
      CUDA_TRY(cudaMemsetAsync(static_cast<char*>(ws) + kErrBytes, 0, kSyncBytes, s),
               "clear synchronisation area");
    CUDA_TRY(cudaStreamSynchronize(s), "stream synchronise");
  }
  if (h & DEVERR_TIMEOUT)
    return fail(ADADSF_ERR_DEVICE_TIMEOUT, "a kernel gave up waiting on a barrier (error word %d)", h);
  if (h & DEVERR_INDEX)
    return fail(ADADSF_ERR_INVALID_ARG, "a kernel met an out-of-range index (error word %d)", h);
  return ADADSF_OK;
}

adadsf_status adadsf_profile_begin(int max_launches) {
  if (max_launches <= 0 || max_launches > (1 << 20))
    return fail(ADADSF_ERR_INVALID_ARG, "max_launches out of range");
  std::lock_guard<std::mutex> lk(g_prof.mu);
  if (g_prof.on) return fail(ADADSF_ERR_INVALID_ARG, "profiling already on");
  while ((int)g_prof.ev.size() < 2 * max_launches) {
    cudaEvent_t e;
    CUDA_TRY(cudaEventCreate(&e), "cudaEventCreate");
    g_prof.ev.push_back(e);
  }
  g_prof.cap = max_launches;
  g_prof.recs.clear();
  g_prof.rec_err.clear();
  g_prof.on = true;
  return ADADSF_OK;
}

int adadsf_profile_end(adadsf_launch_record* out_host, int max) {
  std::lock_guard<std::mutex> lk(g_prof.mu);
  if (!g_prof.on) {
    fail(ADADSF_ERR_INVALID_ARG, "profiling is not on");
    return -1;
  }
  g_prof.on = false;
  if (cudaDeviceSynchronize() != cudaSuccess) {
    fail(ADADSF_ERR_CUDA, "cudaDeviceSynchronize failed");
    return -1;
  }
  const int n = (int)g_prof.recs.size();
  for (int i = 0; i < n && i < max && out_host; ++i) {
    adadsf_launch_record r = g_prof.recs[i];
    float ms = 0.f;
    const cudaError_t e = cudaEventElapsedTime(&ms, g_prof.ev[2 * i], g_prof.ev[2 * i + 1]);
    // failures are reported as negative times: -(1000 + record error) or -(2000 + query error)
    r.ms = g_prof.rec_err[i] ? -(1000.0 + g_prof.rec_err[i]) : (e != cudaSuccess ? -(2000.0 + (int)e) : ms);
    out_host[i] = r;
  }
  return n;
}

const char* adadsf_kernel_name(int kind) {
  static const char* names[ADADSF_KERNEL_COUNT] = {
      "embed", "router", "topk", "positions", "gather_norm", "gemm_qkv", "rope_table", "rope",
      "attention", "gemm_o", "norm2", "gemm_up", "gemm_down", "stats", "final_norm", "copy",
      "linear", "selftest", "gemm_qkv_up", "gemm_o_down", "topk_gather_norm", "decide", "kv_cache", "align"};
  return (kind >= 0 && kind < ADADSF_KERNEL_COUNT) ? names[kind] : "unknown";
}

adadsf_status adadsf_selftest_bounded_wait(void* ws, size_t ws_bytes, int timeout_us, void* stream) {
  TRY(check_ws(ws, ws_bytes, kErrBytes));
  if (timeout_us <= 0 || timeout_us > 2000000)
    return fail(ADADSF_ERR_INVALID_ARG, "timeout_us must be in (0, 2e6]");
  Dev dev;
  TRY(device_info(&dev, stream, ws));
  CUDA_TRY(bounded_wait_selftest(timeout_us, dev), "bounded-wait self-test");
  return ADADSF_OK;
}

}  // extern "C"
