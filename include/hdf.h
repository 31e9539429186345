/*
 * hdf.h — C ABI of the GB300 (sm_103a) HyperDFlash block-drafting library.
 *
 * One draft step is four calls, in the order of the method:
 *   hdf_gated_reduce    Eq. 1 (Sec. 2.2): m-path pre-collapse residual -> [T, d]
 *   hdf_draft_block     Sec. 2.1/2.3: conditioning projection + one non-causal
 *                       block forward of [anchor, mask x (B-1)] over the context
 *   hdf_lm_head_argmax  Sec. 2.3: logits, argmax drafts, optional log-softmax
 *                       at temperature T_KD (the q^{T_KD} of Eq. 2)
 *   hdf_accept_len      Sec. 3.4: accepted-prefix length of each block
 * hdf_accept_sample is the temperature-1 (sampling) form of step 4, and
 * hdf_kl_distill the training-time distillation target (Eq. 2, Sec. 2.3).
 * hdf_ctx_append + hdf_draft_block_cached split step 2 for serving: the
 * context projection of each accepted token runs once, into a K/V cache;
 * hdf_draft_round does both in one call.  hdf_draft_loss is the training
 * objective of Eq. 3, hdf_gated_reduce_backward the gradient of Eq. 1 with
 * respect to W_f and b, and hdf_fc_reduce the generic fc collapse the paper
 * compares against (and falls back to for unequal widths, Sec. 2.2).
 *
 * Conventions shared by every call
 *   - All tensor arguments are DEVICE pointers owned by the caller, row-major,
 *     16-byte aligned, densely packed unless a stride argument says otherwise.
 *     The library keeps no pointer after a call returns.
 *   - The library allocates nothing.  Scratch comes from a caller workspace
 *     (256-byte aligned) whose size the matching *_workspace_size() returns
 *     (hdf_lm_head_argmax_static uses a fixed device array of the library
 *     instead).
 *   - Calls may come from several host threads, and one process may drive
 *     several GPUs: the per-device set-up the library does on first use
 *     (kernel shared-memory limits, occupancy answers) is guarded by a lock.
 *   - Every call is asynchronous on the caller's CUDA stream (a cudaStream_t
 *     passed as hdf_stream_t; NULL = legacy default stream).  No call
 *     synchronises, and there is no host fallback: if the CUDA kernels cannot
 *     run the call returns HDF_ERR_CUDA.  hdf_draft_block (without a trace)
 *     runs its context projection on a second stream that the library keeps
 *     per host thread and device (created on first use, with a few events):
 *     forked from the caller's stream by an event when the call starts and
 *     joined back into it before the call's later kernels, so the call's work
 *     is still ordered after earlier work on the caller's stream and before
 *     later work, and the pair captures into one CUDA graph.
 *   - Arguments are validated on the host before any launch; a rejected call
 *     launches nothing and returns a non-zero status.  hdf_last_error() gives
 *     a human-readable reason (thread-local, valid until the next call).
 *   - dtype is HDF_BF16 (bf16 storage, fp32 accumulation) or HDF_F32 (fp32
 *     storage; GEMMs then run on the tensor cores' tf32 mode).
 *   - Kernels that wait on hardware barriers give up after a bounded time and
 *     record HDF_ERR_DEVICE_CHECK in a device status word that
 *     hdf_device_status() reads; they never trap.  Bounds that depend on
 *     device data (cache lengths) are checked the same way: the access is
 *     skipped and the status word records it.
 */
#ifndef HDF_H
#define HDF_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define HDF_API __attribute__((visibility("default")))
#else
#define HDF_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* hdf_stream_t; /* ABI-identical to cudaStream_t */

enum hdf_status {
  HDF_OK = 0,
  HDF_ERR_INVALID_ARG = 1,  /* null pointer, non-finite or out-of-range scalar */
  HDF_ERR_SHAPE = 2,        /* sizes inconsistent or outside the supported set */
  HDF_ERR_DTYPE = 3,        /* unknown dtype */
  HDF_ERR_ALIGNMENT = 4,    /* a pointer is not 16-byte aligned */
  HDF_ERR_WORKSPACE = 5,    /* workspace missing, misaligned or too small */
  HDF_ERR_CUDA = 6,         /* a CUDA runtime/driver call or launch failed */
  HDF_ERR_UNSUPPORTED = 7,  /* valid request this build does not implement */
  HDF_ERR_DEVICE_CHECK = 8  /* a kernel's bounded wait gave up, or a device-side
                               bound check failed (device word) */
};

enum hdf_dtype { HDF_F32 = 0, HDF_BF16 = 1 };

/* Version of this ABI (major * 100 + minor). */
HDF_API int hdf_version(void);
/* Static string for a status code. */
HDF_API const char* hdf_status_str(int status);
/* Detail of the last failed call on this host thread ("" if none). */
HDF_API const char* hdf_last_error(void);
/* Synchronises the current device, returns the device status word
 * (HDF_OK or HDF_ERR_DEVICE_CHECK) and clears it when reset != 0. */
HDF_API int hdf_device_status(int reset);

/* ------------------------------------------------------------------------
 * (1) Inherited HC-Gate reducer — Eq. 1 and the paragraph after it (Sec. 2.2)
 *
 *   r_t     = (mean_{m*d}(vec H_t ^2) + rms_eps)^(-1/2)
 *   g_tj    = gate_scale * r_t * (W_f vec H_t)_j + b_j
 *   alpha_tj= sigmoid(g_tj) + gate_offset        (independent per-path gates)
 *   y_t     = sum_j alpha_tj * H^_tj
 * with H^_tj = H_tj, or, when path_norm_w != NULL, the drafter-side per-path
 * RMSNorm H_tj * (mean_d(H_tj^2) + path_norm_eps)^(-1/2) * path_norm_w[j].
 * vec() is path-major: vec(H_t)[p*d + e] = H_t[p][e].
 *
 *   H            [n_tokens, m, d]  dtype     pre-collapse residual
 *   Wf           [m, m*d]          dtype     gate weight (RMSNorm weight folded in)
 *   b            [m]               fp32      gate bias
 *   path_norm_w  [m, d] dtype or NULL
 *   alpha_override [n_tokens, m] fp32 or NULL: use these gates instead
 *                (alpha = 1/m gives mean pooling, one-hot selects a path);
 *                Wf and b are then not read and may be NULL
 *   y            [n_tokens, d]     dtype     output (may not alias H)
 *   alpha_out    [n_tokens, m] fp32 or NULL: the gates actually applied
 * Supported: 1 <= m <= 8 (m in {1,2,3,4,8}), d % 8 == 0 (bf16) or d % 4 == 0
 * (fp32), d <= 16384, n_tokens >= 0 (0 launches nothing).
 * ---------------------------------------------------------------------- */
HDF_API int hdf_gated_reduce(const void* H, int dtype, int64_t n_tokens, int m, int d,
                     const void* Wf, const float* b,
                     float rms_eps, float gate_scale, float gate_offset,
                     const void* path_norm_w, float path_norm_eps,
                     const float* alpha_override,
                     void* y, float* alpha_out, hdf_stream_t stream);

/* hdf_gated_reduce with an explicit kernel choice for this call only (no
 * state is kept between calls, so no call can change which kernel, and so
 * which fp32 summation order, another call uses).  The paper has no
 * counterpart: it is a tuning and test hook.  All kernels compute Eq. 1 and
 * agree within fp32 summation order.
 *   HDF_REDUCE_AUTO     what hdf_gated_reduce runs: the tile kernel for m = 4
 *                       where it applies (below), the general kernel
 *                       otherwise, whatever n_tokens is, so that a token's y
 *                       does not depend on how many tokens share the call
 *   HDF_REDUCE_GENERAL  one CTA streams whole tokens and re-reads them from L2
 *                       for the weighted sum (every dtype and option)
 *   HDF_REDUCE_CLUSTER  8-CTA clusters split d, keep W_f slices in shared
 *                       memory and exchange the gate partials of small token
 *                       batches over distributed shared memory
 *   HDF_REDUCE_TILE     persistent clusters of 4 (or, for wide slices, 8)
 *                       CTAs split d over tiles of 16 or 32 tokens, gate dots
 *                       on the tensor cores, one exchange per tile; the
 *                       geometry depends on m and d only
 * CLUSTER and TILE need bf16, m in {1,2,4} and neither alpha_override nor
 * path_norm_w.  CLUSTER also needs d % 512 == 0; TILE needs d a multiple of
 * 64 times its cluster size, a whole number of its 4 box phases per tile and
 * a tile slice that fits its shared memory (for m = 4: every d % 256 == 0 up
 * to 9728, and some wider).  The general kernel runs otherwise.  Another
 * kernel value returns HDF_ERR_INVALID_ARG. */
enum { HDF_REDUCE_AUTO = 0, HDF_REDUCE_GENERAL = 1, HDF_REDUCE_CLUSTER = 2, HDF_REDUCE_TILE = 3 };
HDF_API int hdf_gated_reduce_kernel(int kernel, const void* H, int dtype, int64_t n_tokens, int m, int d,
                     const void* Wf, const float* b,
                     float rms_eps, float gate_scale, float gate_offset,
                     const void* path_norm_w, float path_norm_eps,
                     const float* alpha_override,
                     void* y, float* alpha_out, hdf_stream_t stream);

/* Gradient of the reducer (Eq. 1) with respect to its trainable gate
 * parameters W_f and b (Table 1's 65K parameters), for the loss
 * L = sum_t dy_t . y_t, with H held fixed (the frozen target's residual),
 * gate_offset not entering, no per-path norm and no gate override:
 *   a_tj   = dy_t . H_tj                                 (dL/dalpha_tj)
 *   dg_tj  = a_tj * sigmoid(g_tj) * (1 - sigmoid(g_tj))  (g_tj as above)
 *   db_j   = sum_t dg_tj
 *   dWf[j] = sum_t gate_scale * r_t * dg_tj * vec(H_t)
 *
 *   H, Wf, b, rms_eps, gate_scale   as in hdf_gated_reduce
 *   dy   [n_tokens, d]  dtype   dL/dy (the upstream gradient)
 *   dWf  [m, m*d]       fp32    out, overwritten (16-byte aligned)
 *   db   [m]            fp32    out, overwritten
 *   ws   caller workspace of hdf_gated_reduce_backward_workspace_size()
 *        bytes (256-byte aligned; 0 bytes when n_tokens == 0)
 * Every sum runs in a fixed order: the result is bitwise reproducible.
 * Same m, d and dtype support as hdf_gated_reduce; n_tokens == 0 writes
 * zero gradients.  The paper trains the reducer but prints no backward; this
 * is the chain rule of Eq. 1. */
HDF_API size_t hdf_gated_reduce_backward_workspace_size(int64_t n_tokens, int m, int d, int dtype);
HDF_API int hdf_gated_reduce_backward(const void* H, int dtype, int64_t n_tokens, int m, int d,
                              const void* Wf, const float* b, float rms_eps, float gate_scale,
                              const void* dy, float* dWf, float* db, void* ws, size_t ws_bytes,
                              hdf_stream_t stream);

/* Generic fc reducer of vanilla DFlash (Sec. 2.2, Table 1 "generic fc"),
 * the comparison path and the fallback the paper names for when the
 * reducer's assumptions fail (a source other than the pre-collapse residual,
 * or a drafter width d_out that differs from the target width d_in):
 *   y_t = W_fc vec(H_t),   H [n_tokens, m, d_in], W_fc [d_out, m*d_in],
 *   y [n_tokens, d_out], all dtype; vec() path-major as in Eq. 1.
 * Needs d_out % 128 == 0 and m * d_in * sizeof(dtype) % 16 == 0.  Runs on the
 * tcgen05 GEMM (fp32 accumulation; tf32 inputs for HDF_F32).  Workspace:
 * hdf_fc_reduce_workspace_size() (currently 0 bytes). */
HDF_API size_t hdf_fc_reduce_workspace_size(int64_t n_tokens, int m, int d_in, int d_out, int dtype);
HDF_API int hdf_fc_reduce(const void* H, int dtype, int64_t n_tokens, int m, int d_in, int d_out,
                  const void* W_fc, void* y, void* ws, size_t ws_bytes,
                  hdf_stream_t stream);

/* ------------------------------------------------------------------------
 * (2) Drafter block forward — anchor-plus-mask block input (Sec. 2.1),
 *     conditioning on the reduced pre-collapse residual (Sec. 2.1/2.2),
 *     block slot k predicts the token at a+k (Sec. 2.3).
 *
 * For every sequence i with context rows ctx[cu_ctx[i] .. cu_ctx[i+1]):
 *   c      = RMSNorm_{ctx_norm}(ctx)
 *   h      = [embed[anchor_i]; mask_vec x (B-1)]          (fp32 residual)
 *   per layer:
 *     K_c  = RoPE(c W_k^T, t),  V_c = c W_v^T             (t = 0 .. T_i-1)
 *     x    = RMSNorm_{attn_norm}(h)
 *     Q, K_b, V_b = RoPE(x W_q^T), RoPE(x W_k^T), x W_v^T (positions T_i + k)
 *     O    = softmax(Q [K_c; K_b]^T / sqrt(hd)) [V_c; V_b] per head, no mask
 *     h   += O W_o^T
 *     x    = RMSNorm_{mlp_norm}(h)
 *     h   += (silu(x W_g^T) * (x W_u^T)) W_d^T
 *   h_out  = RMSNorm_{final_norm}(h)
 * RoPE turns pairs (2i, 2i+1) of each head by pos * theta^(-2i/hd), using the
 * caller's tables from hdf_rope_table().  All RMSNorms use shape.norm_eps.
 * bf16 storage points: c, K_c, V_c, x, Q, K_b, V_b, O, silu(.)*(.), h_out.
 * ---------------------------------------------------------------------- */
typedef struct {
  const void* attn_norm; /* [d] */
  const void* wq;        /* [d, d]  (out, in) */
  const void* wk;        /* [d, d] */
  const void* wv;        /* [d, d] */
  const void* wo;        /* [d, d] */
  const void* mlp_norm;  /* [d] */
  const void* wg;        /* [F, d] */
  const void* wu;        /* [F, d] */
  const void* wd;        /* [d, F] */
} hdf_layer_weights;

typedef struct {
  const void* embed;       /* [V, d] */
  const void* mask_vec;    /* [d]   the learned mask-token vector */
  const void* ctx_norm;    /* [d] */
  const void* final_norm;  /* [d] */
  const float* rope_cos;   /* [rope_max_pos, head_dim/2] fp32 */
  const float* rope_sin;   /* [rope_max_pos, head_dim/2] fp32 */
  int64_t rope_max_pos;    /* must exceed max_ctx + block - 1 */
  const hdf_layer_weights* layers; /* HOST array of n_layers entries */
} hdf_drafter_weights;

typedef struct {
  int dtype;       /* HDF_BF16 or HDF_F32, for weights and activations */
  int batch;       /* sequences */
  int block;       /* B: anchor + B-1 mask slots, 2..16 */
  int d;           /* hidden width, d % 128 == 0 */
  int n_heads;     /* n_heads * head_dim == d */
  int head_dim;    /* 64 or 128 */
  int ffn;         /* SwiGLU width F, F % 64 == 0 */
  int vocab;       /* V (embedding rows) */
  int n_layers;    /* >= 1 */
  int max_ctx;     /* upper bound on every T_i (host-side grid sizing) */
  int64_t n_ctx;   /* sum of T_i == cu_ctx[batch] */
  float norm_eps;  /* RMSNorm epsilon */
} hdf_draft_shape;

/* Optional per-stage timing: events[k] (cudaEvent_t) is recorded on the
 * stream before stage k and events[last] after the final stage, so
 * n_events = 3 + HDF_DRAFT_STAGES_PER_LAYER * n_layers (or pass NULL).
 * Stages: context norm, then per layer {context K/V GEMM, block
 * norm (+embedding), QKV GEMM, attention (+combine), O GEMM, MLP norm,
 * gate/up GEMM, down GEMM}, then the final norm.  With a trace every stage
 * runs on the caller's stream, in this order (no second stream). */
#define HDF_DRAFT_STAGES_PER_LAYER 8
typedef struct {
  void* const* events;
  int n_events;
} hdf_trace;

HDF_API size_t hdf_draft_block_workspace_size(const hdf_draft_shape* shape);

/* Where hdf_draft_block leaves its intermediates in the caller's workspace:
 * byte offsets from the workspace start (256-byte aligned), for inspecting a
 * call stage by stage.  Once the call has completed on its stream, and until
 * the workspace is reused, the regions hold (M = batch * block, last = the
 * last layer):
 *   c          [n_ctx, d] dtype  RMSNorm_{ctx_norm}(ctx)
 *   k_ctx      [n_ctx, d] dtype  K_c of the last layer (RoPE applied)
 *   v_ctx      [n_ctx, d] dtype  V_c of the last layer
 *   h          [M, d]     fp32   the residual after the last layer, before the final norm
 *   x          [M, d]     dtype  RMSNorm_{mlp_norm}(h) of the last layer (the MLP input)
 *   q, k_blk, v_blk [M, d] dtype Q, K_b (RoPE applied) and V_b of the last layer
 *   o          [M, d]     dtype  the attention output of the last layer
 *   act        [M, F]     dtype  silu(x W_g^T) * (x W_u^T) of the last layer
 *   total      bytes of the workspace (hdf_draft_block_workspace_size)
 * With shape->n_ctx = 0 the same holds for hdf_draft_block_cached (c, k_ctx
 * and v_ctx are then empty).  The paper has no counterpart: this exists so
 * that each stage can be checked against a reference fed the previous
 * stage's output.  Returns a status like hdf_draft_block's shape check. */
typedef struct {
  size_t c, k_ctx, v_ctx, h, x, q, k_blk, v_blk, o, act, total;
} hdf_draft_workspace_layout;
HDF_API int hdf_draft_block_workspace_layout(const hdf_draft_shape* shape, hdf_draft_workspace_layout* out);
HDF_API int hdf_draft_block(const hdf_drafter_weights* w, const hdf_draft_shape* shape,
                    const void* ctx,        /* [n_ctx, d] dtype (y of Eq. 1) */
                    const int32_t* cu_ctx,  /* [batch + 1] prefix sums of T_i */
                    const int32_t* anchor,  /* [batch] anchor token ids */
                    void* h_out,            /* [batch * block, d] dtype */
                    void* ws, size_t ws_bytes,
                    const hdf_trace* trace, /* NULL: no timing events */
                    hdf_stream_t stream);

/* ------------------------------------------------------------------------
 * (2') Incremental form of step 2 for serving.  In the formula above, the
 *     context keys and values of row t of sequence i depend only on that
 *     row's reduced state and on t:  K_c[t] = RoPE(c_t W_k^T, t),
 *     V_c[t] = c_t W_v^T.  The pre-collapse residual of an accepted token
 *     never changes (Sec. 1: it is stored once, for MTP).  So a serving loop
 *     keeps K_c and V_c of every layer in a cache and, each round, projects
 *     only the tokens accepted since the last round.
 *
 *   hdf_ctx_append          c = RMSNorm_{ctx_norm}(ctx_new), then per layer
 *                           writes K_c, V_c of the new rows at positions
 *                           len[i] .. len[i] + n_i - 1 of sequence i, then
 *                           len[i] += n_i
 *   hdf_draft_block_cached  the block forward of step 2 (same formula, same
 *                           h_out), with T_i = len[i] and K_c, V_c read from
 *                           the cache instead of projected from ctx
 *
 * Appending the rows of a context in any number of rounds and then calling
 * hdf_draft_block_cached gives exactly (bit for bit) the hdf_draft_block
 * output for the whole context, when both use the same shape.max_ctx: every
 * row is projected by the same kernel with the same reduction order, and
 * the attention splits the keys the same way.
 * ---------------------------------------------------------------------- */
typedef struct {
  void* k;       /* [n_layers, batch, capacity, d] dtype: K_c of each layer (RoPE applied) */
  void* v;       /* [n_layers, batch, capacity, d] dtype: V_c of each layer */
  int32_t* len;  /* [batch] DEVICE: rows held per sequence (T_i); the caller
                    zeroes it for a new sequence, hdf_ctx_append advances it */
  int capacity;  /* rows reserved per sequence, >= 1 */
} hdf_ctx_cache;

/* ctx_new [n_ctx, d] dtype: reduced states (y of Eq. 1) of the new rows,
 *         grouped by sequence: rows cu_new[i] .. cu_new[i+1] of sequence i.
 * cu_new  [batch + 1] DEVICE int32, non-decreasing, cu_new[0] = 0.
 * shape.n_ctx is the host's row count of ctx_new; rows at or past
 * cu_new[batch] (<= n_ctx) are skipped, so one captured CUDA graph serves
 * rounds with any number of accepted tokens.  shape.max_ctx is unused.
 * A row whose position would reach cache->capacity is not written: len[i]
 * stops at capacity and HDF_ERR_DEVICE_CHECK is recorded in the device
 * status word (hdf_device_status).  Requires rope_max_pos >= capacity.
 * Workspace: hdf_ctx_append_workspace_size(shape). */
HDF_API size_t hdf_ctx_append_workspace_size(const hdf_draft_shape* shape);
HDF_API int hdf_ctx_append(const hdf_drafter_weights* w, const hdf_draft_shape* shape,
                           const void* ctx_new, const int32_t* cu_new, const hdf_ctx_cache* cache,
                           void* ws, size_t ws_bytes, hdf_stream_t stream);

/* Block forward over the cached context.  shape.max_ctx bounds every len[i]
 * (it sizes the attention split; <= cache->capacity); shape.n_ctx is unused.
 * A len[i] above max_ctx is a contract violation: the keys past max_ctx are
 * not attended and HDF_ERR_DEVICE_CHECK is recorded.  Rows of the cache at
 * or past len[i] may hold anything (they are never read into a result).
 * Requires rope_max_pos >= max_ctx + block.  trace: as for
 * hdf_draft_block (the context-norm and context-K/V stages are empty).
 * Workspace: hdf_draft_block_cached_workspace_size(shape). */
HDF_API size_t hdf_draft_block_cached_workspace_size(const hdf_draft_shape* shape);
HDF_API int hdf_draft_block_cached(const hdf_drafter_weights* w, const hdf_draft_shape* shape,
                                   const hdf_ctx_cache* cache, const int32_t* anchor, void* h_out,
                                   void* ws, size_t ws_bytes, const hdf_trace* trace,
                                   hdf_stream_t stream);

/* One serving round: hdf_ctx_append of the new rows followed by
 * hdf_draft_block_cached, with the same results bit for bit (h_out, the
 * cache rows and len).  The block's input norm and Q / K_b / V_b projection
 * of the first layer do not depend on the new rows, so they run on a second
 * stream beside the append (their RoPE positions are len[i] + n_i, the
 * lengths the append leaves); the lengths are advanced once both are done,
 * before the first attention.  Run serially when stage times are traced.
 * shape.n_ctx is the host's row count of ctx_new (as for hdf_ctx_append);
 * shape.max_ctx bounds every len[i] after the append (as for
 * hdf_draft_block_cached).  Requires rope_max_pos >= capacity and
 * >= max_ctx + block.  Errors as the two calls.
 * Workspace: hdf_draft_round_workspace_size(shape), 256-byte aligned. */
HDF_API size_t hdf_draft_round_workspace_size(const hdf_draft_shape* shape);
HDF_API int hdf_draft_round(const hdf_drafter_weights* w, const hdf_draft_shape* shape,
                            const void* ctx_new, const int32_t* cu_new, const hdf_ctx_cache* cache,
                            const int32_t* anchor, void* h_out, void* ws, size_t ws_bytes,
                            hdf_stream_t stream);

/* cos/sin tables for the drafter's RoPE: entry [p][i] = cos/sin of
 * p * theta^(-2i/head_dim), computed in fp64 on the device and stored fp32.
 * A per-model constant: build once, pass through hdf_drafter_weights. */
HDF_API int hdf_rope_table(double theta, int head_dim, int64_t max_pos,
                   float* cos_out, float* sin_out, hdf_stream_t stream);

/* ------------------------------------------------------------------------
 * (3) LM head — draft logits z = h W_lm^T (Sec. 2.3), greedy drafts
 *     tok = argmax_v z (lowest index wins ties), optional fp32 log-softmax
 *     of z * inv_temp, the log of q^{T_KD} in Eq. 2 (inv_temp = 1/T_KD).
 *
 *   h           [M, d]  dtype
 *   W_lm        [V, d]  dtype
 *   tok         [M]     int32
 *   zmax        [M]     fp32 or NULL: the maximal logit
 *   logsoftmax  [M, V]  fp32 or NULL
 * Row r = i*B + k of a block: k >= 1 holds draft d_k of sequence i.
 * ---------------------------------------------------------------------- */
HDF_API size_t hdf_lm_head_workspace_size(int64_t M, int d, int64_t V, int dtype);
HDF_API int hdf_lm_head_argmax(const void* h, int dtype, int64_t M, int d,
                       const void* W_lm, int64_t V, float inv_temp,
                       int32_t* tok, float* zmax, float* logsoftmax,
                       void* ws, size_t ws_bytes, hdf_stream_t stream);

/* Same computation and arguments as hdf_lm_head_argmax, but without a
 * workspace argument.  The paper has no counterpart: this entry point exists
 * for callers that cannot hand the library device memory -- for instance a
 * plugin whose host process owns every device allocation through its own
 * pool, or code that runs where no allocator may be called once serving has
 * started.  The scratch lives in a file-scope device array of
 * HDF_LM_HEAD_STATIC_SCRATCH_BYTES that every GPU loading the library keeps
 * until the process exits; the call allocates nothing.
 *   - The first call on a device looks up the array's device address (once
 *     per device, with that device current); make that first call before any
 *     stream capture.
 *   - All calls share the one array and it keeps the last call's contents:
 *     two calls whose kernels overlap on the GPU (different streams, or
 *     different host threads) race and corrupt each other's results.
 *   - A request needing more scratch than the array holds (hdf_lm_head_
 *     workspace_size() above the limit) returns HDF_ERR_WORKSPACE and
 *     launches nothing; use hdf_lm_head_argmax with a workspace then. */
#define HDF_LM_HEAD_STATIC_SCRATCH_BYTES (16u << 20)
HDF_API int hdf_lm_head_argmax_static(const void* h, int dtype, int64_t M, int d,
                       const void* W_lm, int64_t V, float inv_temp,
                       int32_t* tok, float* zmax, float* logsoftmax,
                       hdf_stream_t stream);

/* ------------------------------------------------------------------------
 * (4) Block verification — greedy acceptance (Sec. 1, Sec. 3.4):
 *   accept[i] = max{ n <= n_draft : draft[i][k] == target[i][k] for k < n }
 * draft row i starts at draft + i*draft_stride (elements), likewise target,
 * so the drafts can be read straight out of hdf_lm_head_argmax's tok
 * (draft = tok + 1, draft_stride = B).  tau = mean(accept + 1) counts the
 * bonus token (Table 2 prints tau above the number of drafted steps).
 * 0 <= n_draft <= 47 (HDF_ERR_UNSUPPORTED above: the rows of 128 sequences
 * are staged in 48 KB of shared memory).
 * ---------------------------------------------------------------------- */
HDF_API int hdf_accept_len(const int32_t* draft, int64_t draft_stride,
                   const int32_t* target, int64_t target_stride,
                   int batch, int n_draft, int32_t* accept, hdf_stream_t stream);

/* ------------------------------------------------------------------------
 * (4') Temperature-1 block verification by speculative sampling (the T = 1
 * rows of Tables 2 and 3; the paper uses the standard rule without
 * restating it).  For sequence i:
 *   draft slot k (k = 0, 1, ...) is accepted when u[i][k] / 2^32 < p / q with
 *   p = p_target[i][k][x], q = q_draft[i][k][x], x = draft[i][k], the ratio
 *   one IEEE fp32 division (q = 0 accepts, 0/0 rejects, x outside [0, V)
 *   rejects); the first rejection ends the block:  accept[i] = slots accepted.
 *   next_tok[i] is drawn from norm(max(0, p - q)) at the rejected slot (from p
 *   there if that residual is empty), or from p_target[i][n_draft] (the bonus
 *   slot) when every draft is accepted: the first v whose prefix sum of
 *   floor(w * 2^40) exceeds floor(r[i] * R / 2^32), R the total (exact
 *   integer arithmetic); -1 when the distribution has no weight.
 *   p_target [batch, n_draft + 1, V]  fp32 probabilities (target model, T = 1)
 *   q_draft  [batch, n_draft, V]      fp32 probabilities (drafter)
 *   draft    row i at draft + i*draft_stride (e.g. hdf_lm_head_argmax's tok
 *            + 1 with stride B, or sampled drafts)
 *   u [batch, n_draft], r [batch]     uint32 uniforms, drawn by the caller
 *   1 <= V <= 2^22, n_draft >= 0; batch == 0 launches nothing.
 * Every decision is exact: the same inputs give the same accept / next_tok.
 * ---------------------------------------------------------------------- */
HDF_API int hdf_accept_sample(const float* p_target, const float* q_draft, const int32_t* draft,
                              int64_t draft_stride, const uint32_t* u, const uint32_t* r, int batch,
                              int n_draft, int64_t V, int32_t* accept, int32_t* next_tok,
                              hdf_stream_t stream);

/* ------------------------------------------------------------------------
 * (5) KL distillation target — Eq. 2 (Sec. 2.3):
 *   kl_rows[r] = KL(p_r || q_r) = sum_v p_r(v) * (ls_teacher[r][v] - ls_student[r][v])
 *   kl_mean    = t_kd^2 / rows * sum_r kl_rows[r]
 * where p_r = exp(ls_teacher[r]) and both inputs are log-softmax rows at
 * temperature t_kd, as hdf_lm_head_argmax writes them with inv_temp =
 * 1 / t_kd (teacher: the target LM head on the path-mean residual, which
 * hdf_gated_reduce gives with alpha_override = 1/m; student: the draft
 * logits of the first P block positions).  For a batch of blocks with P rows
 * each, kl_mean is the batch mean of L_KL.  hdf_draft_loss below gives the
 * whole objective of Eq. 3.
 *   ls_teacher, ls_student  [rows, V] fp32 (device), rows >= 0, V >= 1
 *   kl_rows                 [rows] fp32 or NULL
 *   kl_mean                 [1] fp32 or NULL
 *   ws / ws_bytes           scratch of hdf_kl_distill_workspace_size(rows, V)
 *                           bytes, 256-byte aligned
 * Teacher entries of -inf contribute 0; a student -inf where the teacher
 * is finite gives +inf.  The sums run in a fixed order (bitwise
 * reproducible).  rows == 0 launches nothing.
 * ---------------------------------------------------------------------- */
HDF_API size_t hdf_kl_distill_workspace_size(int64_t rows, int64_t V);
HDF_API int hdf_kl_distill(const float* ls_teacher, const float* ls_student, int64_t rows, int64_t V,
                           float t_kd, float* kl_rows, float* kl_mean, void* ws, size_t ws_bytes,
                           hdf_stream_t stream);

/* ------------------------------------------------------------------------
 * (5') Training objective of the drafter — Eq. 3 with Eq. 2 (Sec. 2.3):
 *   L = L_CE + alpha * L_KL
 * over a batch of drafted blocks.  Block i's rows of the student are
 * i*block + k (k = 0 the anchor slot, k >= 1 draft position k, which predicts
 * the token at a + k, as hdf_lm_head_argmax lays them out).
 *   L_CE  mean over every supervised draft position (i, k), k = 1..block-1, of
 *         -log q_k(labels[i][k-1]) at temperature 1 (one-hot supervision)
 *   L_KL  T_KD^2 / P * sum_{k=1..P} KL(p_k^T || q_k^T), averaged over the
 *         blocks, p^T / q^T = softmax(ls / T_KD) of the teacher / student rows
 *   ls_teacher [batch, P, V] fp32  log-softmax at temperature 1 of the
 *              teacher LMHead(h_{a+k-1}), k = 1..P (the target LM head on the
 *              path-mean residual: hdf_gated_reduce with alpha_override = 1/m,
 *              then hdf_lm_head_argmax with inv_temp = 1); NULL when P == 0
 *   ls_student [batch*block, V] fp32  log-softmax at temperature 1 of the
 *              draft logits (hdf_lm_head_argmax, inv_temp = 1)
 *   labels     [batch, block-1] int32 device: true token of each draft
 *              position; < 0 = unsupervised.  A label >= V is a contract
 *              violation: the position is left out and HDF_ERR_DEVICE_CHECK
 *              is recorded in the device status word.
 *   ce_rows    [batch, block-1] fp32 or NULL: per-position CE (NaN where
 *              unsupervised);  kl_rows [batch, P] fp32 or NULL
 *   loss       [3] fp32 device: {L, L_CE, L_KL}; L_CE = 0 when no position
 *              is supervised
 *   ws         hdf_draft_loss_workspace_size(batch, P, V) bytes, 256-byte
 *              aligned (0 bytes when P == 0)
 * Both log-softmax inputs must be normalised at temperature 1: the KL part
 * renormalises them at T_KD in its single pass, the CE part reads one entry.
 * 0 <= P <= block - 1 (the paper supervises P = 2), 2 <= block <= 64,
 * batch * block <= 65535.  Every sum runs in a fixed order (bitwise
 * reproducible); identical teacher and student rows give L_KL = 0 exactly.
 * ---------------------------------------------------------------------- */
HDF_API size_t hdf_draft_loss_workspace_size(int batch, int P, int64_t V);
HDF_API int hdf_draft_loss(const float* ls_teacher, const float* ls_student, const int32_t* labels, int batch,
                           int block, int P, int64_t V, float t_kd, float alpha, float* ce_rows, float* kl_rows,
                           float* loss, void* ws, size_t ws_bytes, hdf_stream_t stream);

#ifdef __cplusplus
}
#endif
#endif /* HDF_H */
