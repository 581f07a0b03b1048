// Host-side declarations shared by the translation units of libadadsf.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>
#include <stddef.h>

namespace adadsf {

enum Dtype : int { kF32 = 0, kBF16 = 1 };
// Bits of the device error word (first int of every workspace).
enum : int { DEVERR_TIMEOUT = 1, DEVERR_INDEX = 2 };
enum Act : int { ACT_NONE = 0, ACT_GELU = 1, ACT_SWIGLU = 2 };

// Epilogue of the projection kernels, applied to the fp32 accumulator
// acc[m][n] of out = A[m,:] . W[n,:]:
//   v = acc + bias[n] + bias2[n]              (either may be null)
//   v = gelu(v)                               (ACT_GELU)
//   v = silu(acc) * acc2                      (ACT_SWIGLU, acc2 from the second weight)
//   v += add_packed[m][n]                     (may be null)
//   v += add_rows[row(m)][n]                  (may be null)
//   out[out_mapped ? row(m) : m][n] = v       row(m) = rows ? rows[m] : m
// A packed row with rows[m] < 0 is skipped: no residual read, no store.
// Score gate (gate_scores set; the gated variant of Sec. 3.4): with
// g = sigmoid(gate_scores[row(m)]) and t = v + add_packed[m][n],
//   out = add_rows[row(m)][n] + g t                                (no gate_base)
//   out = gate_base[row(m)][n] + g (t - gate_base[row(m)][n])      (gate_base; no add_rows)
struct Epilogue {
  int act = ACT_NONE;
  const void* bias = nullptr;
  const void* bias2 = nullptr;   // bf16 tensor-core path only
  const void* add_packed = nullptr;
  int64_t ld_add_packed = 0;
  const void* add_rows = nullptr;
  int64_t ld_add_rows = 0;
  const int32_t* rows = nullptr;
  bool out_mapped = true;
  void* out = nullptr;
  int64_t ld_out = 0;
  // Rotary embedding of the first rope_cols output columns (query and key
  // heads), bf16 tensor-core path only: per head of rope_hd columns, feature
  // i < rope_half pairs with i + rope_half and turns by tab[pos][i], pos =
  // rope_pos ? rope_pos[m] : m % rope_T. Needs rope_half in {4, 8, 16} or a multiple of 32.
  const float2* rope_tab = nullptr;
  const int32_t* rope_pos = nullptr;
  int rope_T = 1, rope_half = 0, rope_hd = 0, rope_cols = 0;
  // Value heads also stored transposed (bf16 tensor-core path): output
  // column n >= vt_col0 of row m = b * vt_seq + j goes to
  // vt[((b * vt_hkv + g) * vt_hd + e) * vt_pad + j], g = (n - vt_col0) / vt_hd,
  // e = (n - vt_col0) % vt_hd.
  void* vt = nullptr;
  int vt_seq = 1, vt_pad = 0, vt_col0 = 0, vt_hd = 0, vt_hkv = 0;
  const float* gate_scores = nullptr;
  const void* gate_base = nullptr;
  int64_t ld_gate_base = 0;
  // RMSNorm of the A rows folded into the projection (its gain already in the
  // weights; bf16 tensor-core path): acc *= rstd[m] before anything else,
  // rstd = 1 / sqrt(sum_j nrm_psum[m * nrm_nps + j] / nrm_d + nrm_eps); for
  // ACT_SWIGLU both accumulators are scaled.
  // nrm_rows (or null): the sums of row m are at nrm_psum[nrm_rows[m] * nrm_nps]
  const float* nrm_psum = nullptr;
  const int32_t* nrm_rows = nullptr;
  int nrm_nps = 0, nrm_d = 0;
  float nrm_eps = 0.f;
  // Sum of squares of each stored 32-column chunk (of the fp32 values before
  // their bf16 rounding): sq_out[m * sq_ld + n / 32] (bf16 path; the next
  // RMSNorm's statistics).
  float* sq_out = nullptr;
  int sq_ld = 0;
  // Eq. 4 partials of each stored 32-column chunk (bf16 path; fp32 values), as float4
  // {x_in . out, |x_in|^2, |out|^2, 0} at cos_out[m * cos_ld + n / 32]; x_in
  // = cos_in[row(m)] when given, else the gathered residual add_rows.
  float4* cos_out = nullptr;
  int cos_ld = 0;
  const void* cos_in = nullptr;
  int64_t ld_cos_in = 0;
  // fp32 output instead of `out` (bf16 path, no residual): out_f32[row][n],
  // leading dimension ld_out (the logits of the output alignment, Eq. 10)
  float* out_f32 = nullptr;
};

// acc = A . W^T (+ A2 . Wk2^T when K2 > 0: a second K source, bf16
// tensor-core path only, K a multiple of 64).
struct GemmArgs {
  const void* A = nullptr;  int64_t lda = 0;   // [M, K]
  const void* W = nullptr;  int64_t ldw = 0;   // [N, K]
  const void* W2 = nullptr;                    // [N, K] (ACT_SWIGLU: W = gate, W2 = up)
  const void* A2 = nullptr;  int64_t lda2 = 0;    // [M, K2]
  const void* Wk2 = nullptr; int64_t ldwk2 = 0;   // [N, K2]
  int64_t M = 0; int N = 0; int K = 0; int K2 = 0;
  // Gathered A (bf16, one K source, no second problem): row m of the product
  // is row a_gather[m] of A, which has a_gather_rows rows (all in range)
  const int32_t* a_gather = nullptr;
  int64_t a_gather_rows = 0;
  Epilogue epi;
  // fp32 scratch for splitting small-M products along K (bf16 path); the
  // split is used only when it fits (gemm_split_scratch_bytes covers every case)
  float* scratch = nullptr;
  size_t scratch_bytes = 0;
  // tile width (N) for this problem when the kernel's is 256: 0 = full, or
  // 128 (half-width tiles; one-CTA kernel)
  int tile_n = 0;
};
// Scratch that lets gemm_bf16 split any small-M product along K.
size_t gemm_split_scratch_bytes();

// Every workspace that carries cross-CTA counters holds them in one area of
// this size right after the device error word (offset 256), whatever the
// shapes of the call: the kernels that count there leave the counters at
// zero, so a workspace zero-filled once stays valid for calls of any shape.
constexpr size_t kSyncBytes = 16384;

struct Dev {
  cudaStream_t stream;
  int* err;          // device error word
  int num_sms;
};

// Tensor map of a row-major bf16 [rows, cols] matrix (leading dimension ld
// elements), box_cols x box_rows boxes, 128-byte swizzle, zero fill.
bool make_tmap_bf16(CUtensorMap* m, const void* ptr, uint64_t rows, uint64_t cols, uint64_t ld,
                    uint32_t box_cols, uint32_t box_rows);

// gemm_tcgen05.cu -- bf16 tensor-core projections (tcgen05 + TMEM + TMA).
cudaError_t gemm_bf16(const GemmArgs& a, const Dev& dev);
// Two independent plain projections (no SwiGLU, router or second K source)
// in one launch.
cudaError_t gemm_bf16_grouped(const GemmArgs& a, const GemmArgs& b, const Dev& dev);
// train.cu -- alignment objective (Eqs. 9-10) and the router gradient.
int train_row_blocks(int64_t n);
cudaError_t align_hidden(int dtype, const void* hs, const void* hd, int64_t n_rows, int d, float* grad,
                         double* partials, double* acc, const Dev& dev);
cudaError_t kl_rows(const float* ls, const float* ld, int64_t n_rows, int n_cls, double* partials, double* acc,
                    const Dev& dev);
cudaError_t router_backward(int dtype, const void* x, const void* y_plain, const int32_t* rows, int64_t M, int d,
                            int h, const void* w1, const void* b1, const void* w2, const void* b2, const float* G,
                            float* du, float* su, float* ds, float* grad, const Dev& dev);
// gemm_simt.cu -- fp32 projections on CUDA cores.
cudaError_t gemm_f32(const GemmArgs& a, const Dev& dev);

// attention.cu -- causal attention among kept tokens, fp32 storage.
cudaError_t attention(int dtype, const void* qkv, int64_t ld_qkv, void* out, int64_t ld_out, int B,
                      int K, int n_heads, int n_kv_heads, int head_dim, const Dev& dev);

// attention_tc.cu -- bf16 attention on tcgen05; V enters transposed:
// vt[((b * Hkv + g) * hd + e) * vt_pad(K) + j].
int vt_pad(int K);
cudaError_t vt_from_qkv(const void* qkv, int64_t ld_qkv, int col0, int B, int K, int Hkv, int hd,
                        void* vt, const Dev& dev);
cudaError_t attention_tc(const void* qkv, int64_t ld_qkv, const void* vt, void* out, int64_t ld_out,
                         int B, int K, int n_heads, int n_kv_heads, int head_dim, const Dev& dev);

// rowwise.cu
cudaError_t embed(int dtype, const int32_t* ids, int64_t n, const void* table, int vocab, int d,
                  void* out, const Dev& dev);
// out1 = norm1(x[row(m)]), out2 = norm2(x[row(m)]) (out2 may be null); is_rms selects RMSNorm.
cudaError_t gather_norm(int dtype, const void* x, const int32_t* rows, int64_t M, int d,
                        bool is_rms, const void* g1, const void* b1, const void* g2,
                        const void* b2, float eps, void* out1, void* out2, const Dev& dev);
cudaError_t rope_table(float2* tab, int T, int rotary_dim, float theta, const Dev& dev);
cudaError_t rope_apply(int dtype, void* qkv, int64_t M, int64_t ld, int n_heads, int n_kv_heads,
                       int head_dim, int rotary_dim, const int32_t* pos, int T, const float2* tab,
                       const Dev& dev);
cudaError_t router_f32(const float* x, int64_t n, int d, int h, const float* w1, const float* b1,
                       const float* w2, const float* b2, float* scores, const Dev& dev);
cudaError_t topk(const float* scores, int B, int T, int K, int32_t* idx, int32_t* rows,
                 const Dev& dev);
// router_tc.cu -- bf16 router on tcgen05: scores[r] = w2 . SiLU(W1 x[r] + b1) + b2
// for r < rows. sync: the workspace's synchronisation area (kSyncBytes, zero
// before the call and left at zero) and partials: router_partial_bytes() of
// fp32 scratch, both needed to split 128-token tiles along d (either null:
// no split). tsq (or null): tsq[r] = sum of x[r][j]^2 over j < d, fp32, from
// the same loads (the first RMSNorm's statistic of every token).
size_t router_partial_bytes();
cudaError_t router_tc(const void* x, int64_t rows, int d, const void* w1, const void* b1, const void* w2,
                      const void* b2, float* scores, float* tsq, int* sync, float* partials, const Dev& dev);
// Top-K of each sequence's scores fused with gather_norm of the kept rows
// (out rows b K + i, i-th kept position ascending); also writes idx / rows.
cudaError_t select_gather_norm(int dtype, const float* scores, int B, int T, int K, const void* x,
                               int d, bool is_rms, const void* g1, const void* b1, const void* g2,
                               const void* b2, float eps, void* out1, void* out2, int32_t* idx,
                               int32_t* rows, const Dev& dev);
int stats_partials_count(int64_t n_rows);
cudaError_t iota_positions(int32_t* idx, int B, int K, const Dev& dev);
cudaError_t cos_stats(int dtype, const void* a, const void* b, int64_t n_rows, int d, int mode,
                      double* partials, double* acc, const Dev& dev);
cudaError_t bounded_wait_selftest(int timeout_us, const Dev& dev);
// Eq. 4 sums from per-32-column-chunk partials {a.b, |a|^2, |b|^2} ([n_rows][nch]).
cudaError_t cos_stats_chunks(const float4* parts, int64_t n_rows, int nch, int mode, double* partials,
                             double* acc, const Dev& dev);
// fold.cu -- norm gains (and GPT-NeoX norm biases) folded into the projections, in place.
cudaError_t fold_layer_norms(int dtype, bool neox, int d, int qkv, int F, void* w_qkv, void* b_qkv, void* w_up,
                             void* b_up, void* w_gate, void* g1, void* b1, void* g2, void* b2, const Dev& dev);
// Workspace-free variant of cos_stats: partial sums in a fixed device array.
int stats_static_capacity();
cudaError_t cos_stats_static(int dtype, const void* a, const void* b, int64_t n_rows, int d,
                             int mode, double* acc, const Dev& dev);

// decode.cu -- generation with a cache of kept tokens only (see decode.cu).
int decode_splits(int B, int Hkv, int C_max, int num_sms);
cudaError_t kv_fill(int dtype, const void* qkv, int64_t ld, int q, int kvw, int B, int K, int hd,
                    int C_max, void* kc, void* vc, const Dev& dev);
cudaError_t kv_threshold(const float* scores, const int32_t* idx, int B, int T, int K, int32_t* lens,
                         float* thr, const Dev& dev);
cudaError_t cache_header(int32_t* hdr, int T, int C_max, int L, int B, const Dev& dev);
// Keep decision of each new token (one per sequence) at one layer (decode.cu).
cudaError_t decode_decide(const float* scores, const float* thr, const int32_t* hdr, int B, int C_max,
                          int32_t* rows, int32_t* pos, int32_t* kept_out, const Dev& dev);
// Keep decision of each new token (one per sequence) at one layer, fused with
// the norm(s) of the B new rows (rowwise.cu).
cudaError_t decide_norm(int dtype, const void* x, int B, int d, bool is_rms, const void* g1, const void* b1,
                        const void* g2, const void* b2, float eps, void* out1, void* out2, const float* scores,
                        const float* thr, const int32_t* hdr, int C_max, int32_t* rows, int32_t* pos,
                        int32_t* kept_out, const Dev& dev);
cudaError_t decode_attention(int dtype, const void* qkv, int64_t ld, int Hq, int Hkv, int hd, const void* kc,
                             const void* vc, const int32_t* lens, int C_max, int B, float* part_o,
                             float2* part_ml, void* out, int64_t ld_out, const Dev& dev);
// Rotary embedding of the decode rows fused with the cache append (rotary_dim 0: append only).
cudaError_t rope_append(int dtype, void* qkv, int64_t ld, int Hq, int Hkv, int hd, int rotary_dim, int B,
                        const int32_t* rows, const int32_t* pos, const float2* tab, int32_t* lens, int C_max,
                        void* kc, void* vc, const Dev& dev);
cudaError_t decode_advance(int32_t* hdr, const Dev& dev);

}  // namespace adadsf
