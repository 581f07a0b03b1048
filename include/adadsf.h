/*
 * adadsf.h -- C ABI of the GB300 depth-sparse forward of AdaDSF
 * ("Adaptive Depth Sparse Framework: Similarity-Driven Resource Allocation
 *  for Pre-Trained LLMs").
 *
 * Conventions shared by every entry point
 *  - Pointers named *_dev are device pointers (CUDA global memory of the
 *    current device); pointers named *_host are host pointers. The caller owns
 *    all memory. No entry point allocates or frees device memory; scratch
 *    space comes from a caller-provided workspace (ws, ws_bytes), which must
 *    be zero-filled before its first use (its first 256 bytes hold the device
 *    error word, which must start at zero).
 *  - Device pointers must be 16-byte aligned; the workspace 256-byte aligned.
 *  - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *    stream). Every device entry point only enqueues work on that stream
 *    (adadsf_decode_step also on a stream of its own that it joins back into
 *    it) and returns without synchronising; results are ready once the
 *    stream is.
 *  - Tensors are dense row-major. Weights are [out_features, in_features]
 *    (the torch.nn.Linear layout); the fused QKV weight stacks the query
 *    rows, then the key rows, then the value rows.
 *  - Activations and weights are stored in cfg->dtype (fp32 or bf16);
 *    accumulation, norms, softmax and residual additions run in fp32 with one
 *    rounding per stored tensor. Router scores are fp32. Indices are int32.
 *  - Errors: every call returns an adadsf_status; on failure nothing was
 *    enqueued (argument errors are detected before the first launch) unless
 *    the status is ADADSF_ERR_CUDA. adadsf_last_error() gives a readable
 *    message for the calling thread. No C++ exception crosses this boundary.
 *  - Kernels that wait on barriers give up after a bounded time, record the
 *    fact in a device error word at the start of the workspace and return;
 *    adadsf_sync_check() reports it as ADADSF_ERR_DEVICE_TIMEOUT.
 */
#ifndef ADADSF_H
#define ADADSF_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  ADADSF_OK = 0,
  ADADSF_ERR_INVALID_ARG = 1,
  ADADSF_ERR_UNSUPPORTED = 2,
  ADADSF_ERR_CUDA = 3,
  ADADSF_ERR_WORKSPACE_TOO_SMALL = 4,
  ADADSF_ERR_DEVICE_TIMEOUT = 5
} adadsf_status;

typedef enum { ADADSF_F32 = 0, ADADSF_BF16 = 1 } adadsf_dtype;

/* GPT-NeoX: out = x + Attn(LN1 x) + MLP(LN2 x), LayerNorm, exact-GELU MLP,
 *           biases on every projection.
 * Qwen2.5:  h = x + Attn(RMS1 x); out = h + MLP(RMS2 h), RMSNorm, SwiGLU MLP,
 *           bias on the QKV projection only. */
typedef enum { ADADSF_ARCH_NEOX = 0, ADADSF_ARCH_QWEN = 1 } adadsf_arch;

/* Eq. 4 statistic aggregation. TOKEN: acc += {sum_rows cos(a_r, b_r), rows};
 * FLAT: acc += {sum a.b, sum |a|^2, sum |b|^2} over all rows. */
typedef enum { ADADSF_STATS_TOKEN = 0, ADADSF_STATS_FLAT = 1 } adadsf_stats_mode;

/* adadsf_model_cfg.flags.
 * ADADSF_FLAG_GATE_SIGMOID: the score-gated variant of Sec. 3.4 (where the
 * router scores stay on the differentiable path in training), in the
 * Mixture-of-Depths form: a kept row becomes x + sigmoid(s) * delta, s its router score, delta
 * the layer's whole residual update (inside the layer nothing changes).
 * Without it (default) scores only select and kept rows get x + delta, so
 * K == T is exactly the dense layer. With it the router runs even when
 * K == T. */
#define ADADSF_FLAG_GATE_SIGMOID 1u
/* ADADSF_FLAG_FOLDED_NORMS: every layer's norm gains are 1 and (GPT-NeoX)
 * norm biases 0, their values folded into the projections that read the
 * normed rows (what adadsf_fold_norms leaves). The layers may then apply a
 * norm's row scale inside those projections instead of a separate pass
 * (bf16 Qwen: the post-attention RMSNorm of at most 128 rows, as in a decode
 * step). With unfolded weights the flag gives wrong results. */
#define ADADSF_FLAG_FOLDED_NORMS 2u
/* ADADSF_FLAG_GATHERED_QKV (with ADADSF_FLAG_FOLDED_NORMS; bf16 Qwen layers
 * that keep K < T tokens of more than 32 rows per SM): the first RMSNorm runs
 * inside the QKV projection. The router also sums the squares of every token
 * row it reads, the projection loads the kept rows of x by row-gather copies
 * (four rows per copy) instead of reading a gathered, normed copy, and its
 * epilogue scales each row by 1 / rms. Exact up to rounding; off by default
 * because the row gathers feed the tensor cores more slowly than the separate
 * gather + norm pass costs (at the Qwen2.5-7B shape the QKV projection takes
 * 3.7x its time). Ignored without ADADSF_FLAG_FOLDED_NORMS. */
#define ADADSF_FLAG_GATHERED_QKV 4u

/* adadsf_alloc_ratios flags */
#define ADADSF_ALLOC_RAW 1u      /* return Eq. 8 unclamped (ratios may exceed 1) */
#define ADADSF_ALLOC_ROUND 2u    /* K = round(r T) instead of floor(r T) */

typedef struct {
  int32_t d;             /* hidden size */
  int32_t n_heads;       /* query heads */
  int32_t n_kv_heads;    /* key/value heads; divides n_heads */
  int32_t head_dim;      /* 64 or 128 */
  int32_t ffn;           /* MLP width */
  int32_t n_layers;
  int32_t vocab;
  int32_t router_hidden; /* width of the router's hidden layer (64) */
  int32_t arch;          /* adadsf_arch */
  int32_t rotary_dim;    /* leading features of each head that rotate; even */
  float rope_theta;      /* rotary base */
  float norm_eps;
  int32_t dtype;         /* adadsf_dtype */
  int32_t flags;         /* ADADSF_FLAG_* (other bits: ADADSF_ERR_UNSUPPORTED) */
} adadsf_model_cfg;

/* Device pointers to one layer's parameters, all in cfg->dtype.
 * NULL marks a tensor the architecture does not have. Shapes:
 * router_w1 [h,d] router_b1 [h] router_w2 [h] router_b2 [1]   (h = router_hidden)
 * ln1_w, ln1_b, ln2_w, ln2_b [d]        (the *_b are NeoX only)
 * w_qkv [q+2kv, d] b_qkv [q+2kv]        (q = n_heads*head_dim, kv = n_kv_heads*head_dim)
 * w_o [d, q] b_o [d]                    (b_o NeoX only)
 * w_up [ffn, d] b_up [ffn]              (b_up NeoX only)
 * w_gate [ffn, d]                       (Qwen only)
 * w_down [d, ffn] b_down [d]            (b_down NeoX only) */
typedef struct {
  const void *router_w1, *router_b1, *router_w2, *router_b2;
  const void *ln1_w, *ln1_b, *ln2_w, *ln2_b;
  const void *w_qkv, *b_qkv, *w_o, *b_o;
  const void *w_up, *b_up, *w_gate, *w_down, *b_down;
} adadsf_layer_weights;

/* embed [vocab, d]; final_w, final_b [d] (final_b NeoX only);
 * layers: HOST array of n_layers adadsf_layer_weights (pointing to device data). */
typedef struct {
  const void *embed, *final_w, *final_b;
  const adadsf_layer_weights *layers;
} adadsf_model_weights;

/* Message describing the last failure on the calling thread ("" if none). */
const char *adadsf_last_error(void);

/* ------------------------------------------------------------------------
 * Workspace sizes (bytes, multiples of 256). Return 0 when the arguments are
 * invalid (see adadsf_last_error).
 * ---------------------------------------------------------------------- */
/* One sparse layer on (B,T,d) with K kept tokens per sequence. */
size_t adadsf_layer_workspace_size(const adadsf_model_cfg *cfg, int B, int T, int K);
/* The whole model; K_host holds n_layers kept counts. with_stats != 0 adds
 * the room the Eq. 4 statistics pass needs. */
size_t adadsf_model_workspace_size(const adadsf_model_cfg *cfg, int B, int T,
                                   const int32_t *K_host, int with_stats);
/* adadsf_layer_stats on n_rows rows. */
size_t adadsf_stats_workspace_size(int64_t n_rows);

/* ------------------------------------------------------------------------
 * Sec. 3.3, Eq. 4: similarity of a layer's input and output hidden states.
 * x_in_dev, x_out_dev: [n_rows, d] in `dtype`. acc_dev: device fp64 array
 * (2 entries for TOKEN mode, 3 for FLAT, see adadsf_stats_mode) to which this
 * call ADDS its partial sums, so calibration batches, layers' calls and ranks
 * can be accumulated; the order of the additions inside one call is fixed
 * (results are bit-reproducible). Per-row cosine uses
 * a.b / (max(|a|,1e-8) max(|b|,1e-8)) with fp32 row sums.
 * ---------------------------------------------------------------------- */
adadsf_status adadsf_layer_stats(const void *x_in_dev, const void *x_out_dev, int64_t n_rows,
                                 int d, int dtype, int mode, double *acc_dev,
                                 void *ws, size_t ws_bytes, void *stream);

/* ------------------------------------------------------------------------
 * Workspace-free variant of adadsf_layer_stats. The paper has no counterpart:
 * it exists for callers that cannot give the library any device memory of
 * their own -- hosts whose GPU memory is entirely owned by another allocator
 * or a pre-reserved pool, plugins that are handed only their input and
 * output buffers, and latency-critical paths where a cudaMalloc (and the
 * synchronisation it may imply) is not acceptable.
 * Same arguments, semantics and results as adadsf_layer_stats, without
 * (ws, ws_bytes): the per-block partial sums go to a fixed 48 KiB array
 * (2048 slots of three doubles, a file-scope static __device__ array in the
 * library) that every GPU which loads the library holds until the process
 * exits. Nothing is allocated: no cudaMalloc, cudaFree or allocating library
 * call.
 * Set-up: the first call on each device looks up the array's device address
 * (cudaGetSymbolAddress) with that device current and caches it per device
 * ordinal; make that first call before any stream capture. The cached address
 * belongs to the context that was current then: the entry point is not valid
 * after cudaDeviceReset, nor from a second context on the same device.
 * The array is shared by every call and keeps the last call's contents. Each
 * call writes every slot it later reads, so nothing needs clearing, but
 * calls whose kernels overlap on the GPU (other streams, other host threads)
 * race on the array and return wrong sums: serialise them.
 * Limit: n_rows <= 2^31 - 1 (larger returns ADADSF_ERR_UNSUPPORTED before any
 * launch). The reduction's launch rule caps its block count at 2048 for every
 * n_rows, one slot per block, so the 2048 slots always suffice; d has no
 * limit beyond that of adadsf_layer_stats.
 * ---------------------------------------------------------------------- */
adadsf_status adadsf_layer_stats_noalloc(const void *x_in_dev, const void *x_out_dev,
                                         int64_t n_rows, int d, int dtype, int mode,
                                         double *acc_dev, void *stream);

/* ------------------------------------------------------------------------
 * Sec. 3.3, Eq. 4: the similarity s_l of each layer from the partial sums
 * that adadsf_layer_stats / adadsf_sparse_model_forward accumulated (summed
 * over calibration batches and replicas). Host only, pure.
 * acc_host: L blocks laid out as the stats accumulator of `mode` --
 *   TOKEN: {sum of cosines, token count} per layer, s_l = sum / count;
 *   FLAT:  {sum a.b, sum |a|^2, sum |b|^2} per layer,
 *          s_l = a.b / (max(|a|,1e-8) max(|b|,1e-8)).
 * s_out_host[L] receives s_l. A non-positive token count or a non-finite
 * result returns ADADSF_ERR_INVALID_ARG.
 * ---------------------------------------------------------------------- */
adadsf_status adadsf_similarity(const double *acc_host, int L, int mode, double *s_out_host);

/* ------------------------------------------------------------------------
 * Sec. 3.3, Eqs. 5-8: layer-wise retention ratios from the similarity vector,
 * then K_l = floor(r_l T) (Sec. 3.4). Host only, pure, no device work.
 * s_host[L] similarities; t target mean retention in [0,1]; tau > 0; beta > 0.
 * Unless ADADSF_ALLOC_RAW, ratios above 1 are clamped to 1 and the leftover
 * budget is spread over the other layers in proportion to r'_l, repeatedly,
 * so that sum r = t L with every r_l <= 1. K_l = floor(r_l T + 1e-9) clamped
 * to [0,T] (ADADSF_ALLOC_ROUND: nearest). Outputs: r_out_host[L] (may be
 * NULL), K_out_host[L] (may be NULL).
 * ---------------------------------------------------------------------- */
adadsf_status adadsf_alloc_ratios(const double *s_host, int L, double t, double tau, double beta,
                                  int T, unsigned flags, double *r_out_host, int32_t *K_out_host);

/* ------------------------------------------------------------------------
 * Folds one layer's norm parameters into the projections that read the normed
 * rows, IN PLACE (a reparameterisation; the layer computes the same function
 * up to one bf16 rounding of the changed weights): for a norm n(x) g + b
 * feeding W with bias c, W <- W diag(g) and c <- c + W b (GPT-NeoX: ln1 ->
 * w_qkv / b_qkv, ln2 -> w_up / b_up; Qwen: ln1_w -> w_qkv, ln2_w -> w_gate
 * and w_up), then g <- 1 and b <- 0. The tensors of `w` are modified (their
 * pointers are const in the struct; they must be writable device memory).
 * Afterwards the layer may run with ADADSF_FLAG_FOLDED_NORMS. Asynchronous
 * on `stream`. No paper counterpart (an implementation device).
 * ---------------------------------------------------------------------- */
adadsf_status adadsf_fold_norms(const adadsf_model_cfg *cfg, const adadsf_layer_weights *w, void *stream);

/* ------------------------------------------------------------------------
 * Sec. 3.5: the feature-preserving alignment objective, on device.
 * Eq. 9 (adadsf_align_hidden), per row r of n_rows rows of d features
 * (dtype): n_r = || softmax(hs_r) - softmax(hd_r) ||_2, the softmax over the
 * row's features; acc_dev[0] += sum_r n_r, acc_dev[1] += n_rows (a layer's
 * L_hid is their ratio). grad_dev (NULL or fp32 [n_rows, d]) receives
 * d n_r / d hs_r = p (r / n - p . r / n), p = softmax(hs_r), r = p -
 * softmax(hd_r) (zero where n = 0); divide by the row count for the mean's
 * gradient.
 * Eq. 10 (adadsf_align_output): KL(P_dense || P_sparse) per row, P the
 * softmax over n_classes of the logits h W_head^T (w_head_dev [n_classes, d],
 * e.g. the tied embedding); acc_dev[0] += sum of the rows' KL, acc_dev[1] +=
 * n_rows. Logits are fp32 (workspace: adadsf_align_workspace_size(n_rows,
 * n_classes), 8 n_rows n_classes bytes of them: call on row chunks for large
 * vocabularies). bf16 needs d and n_classes multiples of 64.
 * Eq. 11 is L_align + (1/L) sum_l L_hid^(l) of those accumulators.
 * Sums run in a fixed order (bit-reproducible).
 * ---------------------------------------------------------------------- */
size_t adadsf_align_workspace_size(int64_t n_rows, int n_classes);
adadsf_status adadsf_align_hidden(const void *hs_dev, const void *hd_dev, int64_t n_rows, int d, int dtype,
                                  double *acc_dev, float *grad_dev, void *ws, size_t ws_bytes, void *stream);
adadsf_status adadsf_align_output(const void *hs_dev, const void *hd_dev, const void *w_head_dev,
                                  int64_t n_rows, int d, int n_classes, int dtype, double *acc_dev,
                                  void *ws, size_t ws_bytes, void *stream);

/* ------------------------------------------------------------------------
 * Sec. 3.4 (router scores on the differentiable path): the gradient
 * of a loss with respect to one layer's router parameters through the score
 * gate of ADADSF_FLAG_GATE_SIGMOID, where a kept row is y = x + sigmoid(s)
 * delta. The layer input and its other weights are held fixed and the Top-K
 * choice carries no gradient. x_dev [B*T, d]: the layer input; y_plain_dev
 * [B*T, d]: the UNGATED layer's output on the same kept set (delta =
 * y_plain - x on kept rows); rows_dev [n_kept]: the kept rows (b*T +
 * position); grad_y_dev fp32 [B*T, d]: dL/dy (only kept rows are read).
 * grad_out_dev fp32 receives, contiguously, dL/dW1 [router_hidden, d],
 * dL/db1 [router_hidden], dL/dw2 [router_hidden], dL/db2 [1]:
 *   ds = sigmoid'(s) (dL/dy . delta), dw2 = sum ds SiLU(u), db2 = sum ds,
 *   du = ds w2 SiLU'(u), dW1 = sum du x^T, db1 = sum du, u = W1 x + b1.
 * ws: adadsf_router_backward_workspace_size(cfg, n_kept) bytes.
 * ---------------------------------------------------------------------- */
size_t adadsf_router_backward_workspace_size(const adadsf_model_cfg *cfg, int64_t n_kept);
adadsf_status adadsf_router_backward(const adadsf_model_cfg *cfg, const adadsf_layer_weights *w,
                                     const void *x_dev, const void *y_plain_dev, const int32_t *rows_dev,
                                     int64_t n_kept, const float *grad_y_dev, float *grad_out_dev,
                                     void *ws, size_t ws_bytes, void *stream);

/* ------------------------------------------------------------------------
 * Sec. 4.1 (the normalized FLOPs of Tables 1-2): FLOPs of the depth-sparse
 * forward over those of the dense model, per sequence of T tokens. Host
 * only, pure. Counted per layer l: the router on all T tokens when
 * K_host[l] < T (2 flops per multiply-add of W1 and w2), plus the layer on its
 * K_host[l] kept tokens -- the QKV, output and MLP projections (three MLP
 * matrices for Qwen's SwiGLU, two for GPT-NeoX) and causal attention among
 * the kept tokens (2 n_heads head_dim K (K + 1)); divided by n_layers dense
 * layers on T tokens. Embedding, final norm and LM head are the same in both
 * and left out. The paper does not state its counting rules; this is the
 * reading used here. K = T everywhere gives 1. *out_host receives the ratio.
 * ---------------------------------------------------------------------- */
adadsf_status adadsf_normalized_flops(const adadsf_model_cfg *cfg, int T, const int32_t *K_host,
                                      double *out_host);

/* ------------------------------------------------------------------------
 * Sec. 3.4: router scores of every token, w2 . SiLU(W1 x + b1) + b2.
 * x_dev [B*T, d] (cfg->dtype); scores_dev [B*T] fp32. ws: at least 256
 * bytes (the device error word); on the bf16 path, with
 * adadsf_router_select_workspace_size(cfg, 1, 1) bytes or more (zero-filled
 * before first use), tiles of 128 tokens may also be split along d over
 * several CTAs.
 * ---------------------------------------------------------------------- */
adadsf_status adadsf_router_scores(const adadsf_model_cfg *cfg, const adadsf_layer_weights *w,
                                   const void *x_dev, int64_t n_rows, float *scores_dev,
                                   void *ws, size_t ws_bytes, void *stream);

/* ------------------------------------------------------------------------
 * Sec. 3.4: Top-K_i of each sequence's router scores, K_i = K for all.
 * scores_dev [B,T] fp32. Ranking: higher score first, equal scores by lower
 * position, -0.0 equals +0.0, NaN below every number. idx_dev [B,K] int32
 * receives the kept positions in ascending order; rows_dev [B,K] int32 (may
 * be NULL) receives b*T + position. 0 <= K <= T <= 16384.
 * ---------------------------------------------------------------------- */
adadsf_status adadsf_topk_select(const float *scores_dev, int B, int T, int K,
                                 int32_t *idx_dev, int32_t *rows_dev, void *stream);

/* ------------------------------------------------------------------------
 * Sec. 3.4: router scores of every token and the Top-K of each sequence in
 * one call (the router kernel, then the Top-K kernel). x_dev [B*T, d]
 * (cfg->dtype); scores_dev [B*T] fp32 receives the scores; idx_dev [B,K]
 * int32 the kept positions of each sequence in ascending order; rows_dev
 * [B,K] int32 (may be NULL) b*T + position. Same ranking as
 * adadsf_topk_select; 1 <= K <= T <= 16384.
 * ws: adadsf_router_select_workspace_size(cfg, B, T) bytes (the same for
 * every B, T), zero-filled before first use. On the bf16 path the router
 * splits 128-token tiles along d over several CTAs when there are few
 * tiles: arrival counters sit in a fixed area right after the device error
 * word (every completed call leaves them at zero, so one workspace serves
 * calls of any shape, here and in the layer and model forwards; after a
 * device timeout, adadsf_sync_check zeroes them), fp32 partial tiles after
 * it.
 * ---------------------------------------------------------------------- */
size_t adadsf_router_select_workspace_size(const adadsf_model_cfg *cfg, int B, int T);
adadsf_status adadsf_router_select(const adadsf_model_cfg *cfg, const adadsf_layer_weights *w,
                                   const void *x_dev, int B, int T, int K, float *scores_dev,
                                   int32_t *idx_dev, int32_t *rows_dev, void *ws, size_t ws_bytes,
                                   void *stream);

/* ------------------------------------------------------------------------
 * Eq. 2 building block: out = act(x W^T + bias). x_dev [M, k_in],
 * w_dev [n_out, k_in], bias_dev [n_out] or NULL, out_dev [M, n_out], all in
 * `dtype`. act: 0 identity, 1 exact GELU. k_in % 64 == 0, n_out % 64 == 0 for
 * bf16 (tcgen05 tensor-core path), multiples of 4 for fp32. ws: at least 256
 * bytes (the device error word); on the bf16 path any bytes beyond the first
 * 256 may serve as fp32 scratch for splitting a small-M product along K over
 * clusters of CTAs (ADADSF_LINEAR_SPLIT_WS_BYTES allows every such split;
 * with less the split is used only where it fits). ws is owned by the caller
 * and must not be in use by another call in flight.
 * ---------------------------------------------------------------------- */
#define ADADSF_LINEAR_SPLIT_WS_BYTES (256u + 160u * 128u * 256u * 4u)
adadsf_status adadsf_linear(const void *x_dev, const void *w_dev, const void *bias_dev,
                            int64_t M, int n_out, int k_in, int dtype, int act, void *out_dev,
                            void *ws, size_t ws_bytes, void *stream);

/* ------------------------------------------------------------------------
 * Eq. 1 among kept tokens: per sequence b and query head h,
 * softmax(Q K^T / sqrt(head_dim)) V, causal in packed order (which is the
 * original order, as kept positions ascend). qkv_dev [B*K, q+2kv] (rotary
 * already applied), out_dev [B*K, q]; cfg->dtype. Query head h reads kv head
 * h / (n_heads / n_kv_heads). ws: adadsf_attention_workspace_size bytes (bf16
 * keeps the value heads transposed there for the tensor cores).
 * ---------------------------------------------------------------------- */
size_t adadsf_attention_workspace_size(const adadsf_model_cfg *cfg, int B, int K);
adadsf_status adadsf_causal_attention(const adadsf_model_cfg *cfg, const void *qkv_dev, int B,
                                      int K, void *out_dev, void *ws, size_t ws_bytes,
                                      void *stream);

/* ------------------------------------------------------------------------
 * Sec. 3.4: one depth-sparse layer, in place.
 * x_dev [B,T,d]: kept rows become x + delta (delta = the layer's residual
 * update computed on the kept tokens only, causal among them, rotary at
 * their original positions; x + sigmoid(score) delta with
 * ADADSF_FLAG_GATE_SIGMOID); every other row is left untouched (not read
 * back nor written). K == 0 enqueues nothing; K == T runs the dense layer
 * (Top-K skipped; the router too unless the gate is on). idx_out_dev [B,K]
 * int32 and scores_out_dev [B,T] fp32 receive the kept positions and router
 * scores (either may be NULL; with K == T and no gate, scores are not
 * computed and scores_out_dev is ignored).
 * ---------------------------------------------------------------------- */
adadsf_status adadsf_sparse_layer_forward(const adadsf_model_cfg *cfg, const adadsf_layer_weights *w,
                                          void *x_dev, int B, int T, int K, int32_t *idx_out_dev,
                                          float *scores_out_dev, void *ws, size_t ws_bytes,
                                          void *stream);

/* ------------------------------------------------------------------------
 * Sec. 3.2 / 3.4: the depth-sparse model. ids_dev [B,T] int32 -> embedding
 * -> layer l as adadsf_sparse_layer_forward with K_host[l] kept tokens ->
 * final norm -> hidden_out_dev [B,T,d] (cfg->dtype).
 * stats_acc_dev: NULL, or device fp64 [n_layers * 2] (TOKEN mode) to which
 *   the Eq. 4 sums of each layer's (input, output) pair are added (the
 *   calibration pass runs this with K_l = T).
 * idx_out_dev: NULL, or device int32 of B * sum_l K_l entries receiving each
 *   layer's kept positions [B, K_l], layer after layer.
 * Out-of-range token ids read as zero rows and raise the device error word.
 * ---------------------------------------------------------------------- */
adadsf_status adadsf_sparse_model_forward(const adadsf_model_cfg *cfg, const adadsf_model_weights *w,
                                          const int32_t *ids_dev, int B, int T, const int32_t *K_host,
                                          void *hidden_out_dev, double *stats_acc_dev,
                                          int32_t *idx_out_dev, void *ws, size_t ws_bytes,
                                          void *stream);

/* ------------------------------------------------------------------------
 * Autoregressive decode with a cache of kept tokens only. The paper defines
 * the sparse forward over whole sequences (Sec. 3.4) and says nothing about
 * generation; this is a Mixture-of-Depths style reading:
 *  - adadsf_prefill runs adadsf_sparse_model_forward on the prompt (B
 *    sequences of T tokens, K_host[l] kept per layer) and also stores, per
 *    layer l and sequence b, the kept tokens' keys (rotated) and values, their
 *    count, and the keep threshold: the lowest router score the layer kept
 *    (the K-th largest; +inf when K_host[l] == 0). It runs the router on
 *    every layer, dense ones included. idx_out_dev as in
 *    adadsf_sparse_model_forward (NULL or B * sum_l K_l int32).
 *  - adadsf_decode_step takes one new token per sequence (ids_dev [B], at
 *    the position after the last one) through every layer: the router
 *    scores the token's hidden state; if the score is strictly above the
 *    layer's threshold (a tie loses, as the later position loses Top-K ties;
 *    NaN never wins), the token attends to the layer's cached kept tokens and
 *    itself, gets the layer's residual delta (x sigmoid(score) with
 *    ADADSF_FLAG_GATE_SIGMOID) and its key and value join the cache;
 *    otherwise it bypasses the layer unchanged. hidden_out_dev [B, d]
 *    receives the final-normed hidden states; kept_out_dev (NULL or int32
 *    [n_layers][B]) the decisions (1 kept, 0 bypassed).
 * The cache is one caller buffer of adadsf_kv_cache_size bytes (256-byte
 * aligned; C_max = positions it can hold, prompt included): a header with
 * the current position, per-layer counts and thresholds, the rotary table
 * of every position and, per layer, K and V as [B][n_kv_heads][C_max]
 * [head_dim] in cfg->dtype. Decode steps read the position and counts from
 * the cache, so their launch arguments never change (one CUDA graph can
 * replay them). A step whose position reaches C_max, or whose layer's
 * cache is full, sets the device error word (adadsf_sync_check reports
 * ADADSF_ERR_INVALID_ARG) and appends nothing. Prefill needs T < C_max and
 * the workspace of adadsf_model_workspace_size(cfg, B, T, K_host, 0); a
 * decode step adadsf_decode_workspace_size(cfg, B, C_max), and at most 16
 * query heads per key/value head (else ADADSF_ERR_UNSUPPORTED).
 * A decode step runs each layer's router and keep decision on a second
 * stream owned by the library, beside the norm and QKV projection on
 * `stream`. Events fork that stream from `stream` and join it back before
 * the layer's cache append, so the step is complete when `stream` is, and a
 * graph captured from `stream` contains it. The second stream is made on
 * the first decode step enqueued on `stream`; a step captured before any
 * uncaptured step on that stream runs on `stream` alone, with the same
 * results.
 * ---------------------------------------------------------------------- */
size_t adadsf_kv_cache_size(const adadsf_model_cfg *cfg, int B, int C_max);
adadsf_status adadsf_prefill(const adadsf_model_cfg *cfg, const adadsf_model_weights *w,
                             const int32_t *ids_dev, int B, int T, const int32_t *K_host,
                             void *hidden_out_dev, int32_t *idx_out_dev, void *cache_dev,
                             size_t cache_bytes, int C_max, void *ws, size_t ws_bytes, void *stream);
size_t adadsf_decode_workspace_size(const adadsf_model_cfg *cfg, int B, int C_max);
adadsf_status adadsf_decode_step(const adadsf_model_cfg *cfg, const adadsf_model_weights *w,
                                 const int32_t *ids_dev, int B, void *hidden_out_dev,
                                 int32_t *kept_out_dev, void *cache_dev, size_t cache_bytes,
                                 int C_max, void *ws, size_t ws_bytes, void *stream);

/* ------------------------------------------------------------------------
 * Synchronises `stream`, then reads and clears the device error word at the
 * start of `ws`: ADADSF_ERR_DEVICE_TIMEOUT if a kernel gave up waiting,
 * ADADSF_ERR_INVALID_ARG if a kernel met an out-of-range index,
 * ADADSF_ERR_CUDA on a CUDA error, else ADADSF_OK.
 * After a timeout it also zero-fills the synchronisation area that follows
 * the error word (16 KiB of cross-CTA arrival counters, when ws_bytes covers
 * it): a kernel that gave up may have left a counter part-way. A workspace
 * that saw a timeout must pass through this call (or be zero-filled again)
 * before its next use.
 * ---------------------------------------------------------------------- */
adadsf_status adadsf_sync_check(void *ws, size_t ws_bytes, void *stream);

/* ------------------------------------------------------------------------
 * Per-launch timing (diagnostics; no paper counterpart). Between
 * adadsf_profile_begin and adadsf_profile_end every kernel the library
 * launches on a stream that is not being captured is bracketed by a pair of
 * CUDA events on that stream and recorded with its algorithmic work:
 * flops (2 per multiply-add of the dense contractions and of attention) and
 * bytes (each input element read once plus each output element written once,
 * skipped rows excluded). adadsf_profile_end synchronises the device, writes
 * up to `max` records and returns the number of records (or -1 on error).
 * Kinds are the ADADSF_KERNEL_* values; adadsf_kernel_name names them.
 * ---------------------------------------------------------------------- */
typedef enum {
  ADADSF_KERNEL_EMBED = 0, ADADSF_KERNEL_ROUTER, ADADSF_KERNEL_TOPK, ADADSF_KERNEL_POSITIONS,
  ADADSF_KERNEL_GATHER_NORM, ADADSF_KERNEL_GEMM_QKV, ADADSF_KERNEL_ROPE_TABLE, ADADSF_KERNEL_ROPE,
  ADADSF_KERNEL_ATTENTION, ADADSF_KERNEL_GEMM_O, ADADSF_KERNEL_NORM2, ADADSF_KERNEL_GEMM_UP,
  ADADSF_KERNEL_GEMM_DOWN, ADADSF_KERNEL_STATS, ADADSF_KERNEL_FINAL_NORM, ADADSF_KERNEL_COPY,
  ADADSF_KERNEL_LINEAR, ADADSF_KERNEL_SELFTEST,
  ADADSF_KERNEL_GEMM_QKV_UP,   /* GPT-NeoX, bf16: QKV and MLP-up projections in one launch */
  ADADSF_KERNEL_GEMM_O_DOWN,   /* GPT-NeoX, bf16: output + MLP-down projections, one accumulator */
  ADADSF_KERNEL_TOPK_GATHER_NORM, /* Top-K fused with the gather and norms of the kept rows */
  ADADSF_KERNEL_DECIDE,        /* decode: keep decision of each new token (inside the norm launch when the step runs on one stream) */
  ADADSF_KERNEL_KV_CACHE,      /* decode cache: fill (prefill), thresholds, append */
  ADADSF_KERNEL_ALIGN,         /* alignment objective and router gradient (Eqs. 9-10) */
  ADADSF_KERNEL_COUNT
} adadsf_kernel_kind;

typedef struct {
  int32_t kind;    /* adadsf_kernel_kind */
  int32_t dense;   /* 1 if the launch runs on tensor cores (flops-bound) */
  double ms;       /* device time between the bracketing events */
  double flops;    /* algorithmic floating-point operations of the launch */
  double bytes;    /* algorithmic HBM bytes of the launch */
} adadsf_launch_record;

adadsf_status adadsf_profile_begin(int max_launches);
int adadsf_profile_end(adadsf_launch_record *out_host, int max);
const char *adadsf_kernel_name(int kind);

/* Self-test of the bounded-wait path: launches one block that waits on a
 * shared-memory barrier nothing arrives at, gives up after about
 * timeout_us microseconds, records ADADSF_ERR_DEVICE_TIMEOUT in the error
 * word of `ws` and returns, leaving the context usable. No paper counterpart. */
adadsf_status adadsf_selftest_bounded_wait(void *ws, size_t ws_bytes, int timeout_us, void *stream);

#ifdef __cplusplus
}
#endif
#endif /* ADADSF_H */
