// Host-side launch interfaces of the CUDA kernels (internal to libhdf).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace hdf {

// Launches a kernel of the draft path with programmatic dependent launch
// (its prologue may overlap the previous kernel in the stream; the kernel
// calls pdl_wait() before touching that kernel's results) and, when
// cluster_x > 1, as clusters of cluster_x consecutive blocks.
// The launch carries the stream's priority as a launch attribute, so that
// kernels captured into a CUDA graph keep the priority of the stream they
// were issued on.
template <typename... KArgs, typename... Args>
cudaError_t launch_kernel(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                          unsigned cluster_x, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[3];
  unsigned n = 0;
  attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[n].val.programmaticStreamSerializationAllowed = 1;
  ++n;
  int prio = 0;
  if (cudaStreamGetPriority(s, &prio) == cudaSuccess && prio != 0) {
    attr[n].id = cudaLaunchAttributePriority;
    attr[n].val.priority = prio;
    ++n;
  } else {
    cudaGetLastError();
  }
  if (cluster_x > 1) {
    attr[n].id = cudaLaunchAttributeClusterDimension;
    attr[n].val.clusterDim.x = cluster_x;
    attr[n].val.clusterDim.y = 1;
    attr[n].val.clusterDim.z = 1;
    ++n;
  }
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = n;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// Per-device kernel set-up, safe from concurrent host threads.  A process may
// drive several GPUs and call the library from several threads: a kernel's
// dynamic shared-memory limit is set on each device before its first launch
// there (raised if a later launch needs more), and occupancy answers are kept
// per device.  Both live in hdf_api.cu behind one lock.
cudaError_t ensure_smem_limit(const void* kernel, size_t smem, bool nonportable_clusters = false);
// Clusters of `cluster` CTAs (`block` threads, `smem` dynamic bytes each) that
// can be resident at once on the current device; 0 when none fit.  The
// caller sets the kernel's shared-memory limit first.
cudaError_t max_active_clusters(const void* kernel, int block, size_t smem, int cluster, int* n);

// ------------------------------------------------------------ reducer ----
struct ReduceArgs {
  const void* H;
  const void* Wf;
  const float* b;
  const void* path_norm_w;
  const float* alpha_override;
  void* y;
  float* alpha_out;
  long long n_tokens;
  int m, d;
  float rms_eps, gate_scale, gate_offset, path_norm_eps;
  int* status;
};
cudaError_t launch_gated_reduce(const ReduceArgs& a, int dtype, cudaStream_t s);

// Gradient of the reducer with respect to W_f and b (reduce_bwd.cu).
struct ReduceBwdArgs {
  const void* H;      // [N, m, d] dtype
  const void* Wf;     // [m, m*d] dtype
  const float* b;     // [m]
  const void* dy;     // [N, d] dtype: dL/dy
  float* dWf;         // [m, m*d] out
  float* db;          // [m] out
  float* u;           // [N, m] workspace: s * r_t * dg_tj
  float* dg;          // [N, m] workspace: dL/dg_tj
  float* part;        // [splits, m, m*d] workspace: per-split weight-gradient sums
  float* dbpart;      // [splits, m] workspace
  long long n_tokens;
  int m, d;
  float rms_eps, gate_scale;
};
struct ReduceBwdPlan {
  int slices = 1, splits = 1, gate_ctas = 1;  // weight-gradient grid (slices x splits), gate-pass CTAs
  long long tok_per = 0;                       // tokens per split
};
ReduceBwdPlan reduce_bwd_plan(long long n_tokens, int m, int d, int dtype, int n_sm);
cudaError_t launch_gated_reduce_backward(const ReduceBwdArgs& a, int dtype, const ReduceBwdPlan& p, cudaStream_t s);
// bf16 cluster path: box {64, rb, E/64} of the 3-D view {64 elements, tokens,
// 128-byte chunks} of H (128-byte swizzle) that the caller encodes; false
// when the shape or options need the general kernel above.
bool reduce_cluster_box(const ReduceArgs& a, int dtype, unsigned box[3]);
cudaError_t launch_gated_reduce_cluster(const ReduceArgs& a, const CUtensorMap* h_map, cudaStream_t s);
// bf16 tile path: boxes {64, 32, C} and {64, 32, tail} of the 3-D view {64
// elements, tokens, 128-byte chunks} of H (128-byte swizzle) that the caller
// encodes as h_maps[0], h_maps[1]; false when the shape or options need the
// general kernel.
bool reduce_tile_boxes(const ReduceArgs& a, int dtype, unsigned box[3], unsigned tail_box[3]);
cudaError_t launch_gated_reduce_tile(const ReduceArgs& a, const CUtensorMap* h_maps, cudaStream_t s);

// --------------------------------------------------------------- GEMM ----
// D[M, N] = A[M, K] * B[N, K]^T, both operands K-major, loaded by TMA with
// 128-byte swizzle.  An operand may be the row-concatenation of up to three
// tensors (one tensor map each), or (A only) a "pair" whose 64-row halves of
// each 128-row tile come from two tensors at the same row offset.
enum OperandMode { kConcat = 0, kPair64 = 1 };

struct Operand {
  CUtensorMap map[3];
  int rows_per_map;  // kConcat: rows covered by each map (tile-aligned)
  int mode;
};

enum EpiKind {
  kEpiStore = 0,    // rows = tokens, cols = features -> out[seg][row, col]
  kEpiStoreT = 1,   // rows = features, cols = tokens -> out[seg][col, row]
  kEpiResidT = 2,   // resid[col, row] += D  (fp32 residual)
  kEpiSwigluT = 3,  // pair tile: act[col, f] = silu(g) * u
  kEpiLmHeadT = 4,  // rows = vocab, cols = tokens: argmax / sum-exp partials
  kEpiLmHead = 5,   // rows = tokens, cols = vocab: the same partials, one per (column tile, token)
};

struct Epilogue {
  int kind;
  void* out[3];         // segment outputs (dtype of the GEMM)
  int seg_width;        // features per segment
  long long ld;         // row stride of out[] / resid / act, elements
  int rope_mask;        // bit s: RoPE on segment s
  const float* rope_cos;
  const float* rope_sin;
  long long rope_rows;  // positions >= rope_rows are clamped (contract violation)
  int head_dim;
  const int* cu_ctx;    // positions: context rows -> t - cu[b]
  int batch;
  int block;            // block rows: pos = T_b + (j % block)
  int pos_mode;         // 0 none, 1 context rows, 2 block rows (T_b from cu_ctx),
                        // 3 context rows appended to a cache, 4 block rows (T_b = ctx_len[b]),
                        // 5 block rows beside an append (T_b = ctx_len[b] + cu[b+1] - cu[b])
  const int* ctx_len;   // modes 3, 4, 5: rows already in the cache per sequence
  long long cache_cap;  // mode 3: row t of sequence b goes to row b * cache_cap + ctx_len[b] + t - cu[b]
  float* resid;         // kEpiResidT
  // kEpiLmHeadT
  float inv_temp;
  float* logsoftmax;    // [N, M] fp32 or null (stored transposed: token-major)
  float* part_max;      // [tiles_m, N]
  int* part_arg;
  float* part_sum;
  // kEpiStore on CTA pairs with packed output rows (pos_mode 0 or 1): the
  // tile is written by TMA stores through these maps of out[0], out[1]
  // ([rows, seg_width], boxes {64, 128}, 128-byte swizzle) when out_tma != 0
  int out_tma;
  CUtensorMap out_map[2];
};

struct GemmArgs {
  Operand A, B;
  int M, N, K;
  int dtype;            // HDF_BF16 or HDF_F32 (tf32)
  int bn;               // tile width along N: 16, 32, 64, 128 or 256
  int k_splits;         // 1..16 (> 1 needs bn <= 128): the splits of a tile run as one thread-block cluster
  int pre_operand;      // 1: A, 2: B does not depend on earlier kernels (weights) and is loaded
                        // before pdl_wait(); 0: neither
  int group_n;          // raster: n-tiles swept together
  int pair;             // 1: 256 x 256 tiles on CTA pairs (cta_group::2); bf16, bn 256, kEpiStore, no K split
                        // (B maps with 128-row boxes)
  Epilogue epi;
  int* status;
};
cudaError_t launch_gemm(const GemmArgs& g, cudaStream_t s);
int gemm_stages(int dtype, int bn);
// CTAs of the GEMM resident at once in clusters of `cluster` (1..16); -1 when
// the device cannot be asked
int gemm_resident_ctas(int dtype, int bn, int cluster);
size_t gemm_smem_bytes(int dtype, int bn);

// ----------------------------------------------------- small kernels ----
cudaError_t launch_rope_table(double theta, int head_dim, long long max_pos, float* c, float* s,
                              cudaStream_t st);
// y[r] = RMSNorm_w(x[r]) for rows r; x fp32 or dtype, y dtype.
cudaError_t launch_rmsnorm(const void* x, int x_is_f32, const void* w, void* y, int dtype,
                           long long rows, int d, float eps, cudaStream_t s);
// h[i*B + 0] = embed[anchor[i]], h[i*B + k] = mask_vec; x = RMSNorm(h).
cudaError_t launch_embed_norm(const void* embed, const void* mask_vec, const int* anchor,
                              const void* norm_w, float* h, void* x, int dtype, int batch,
                              int block, int d, int vocab, float eps, cudaStream_t s);
cudaError_t launch_accept(const int* draft, long long ds, const int* target, long long ts,
                          int batch, int nd, int* accept, cudaStream_t s);
cudaError_t launch_lm_reduce(const float* part_max, const int* part_arg, const float* part_sum,
                             int tiles, long long M, long long V, float inv_temp, int* tok,
                             float* zmax, float* logsoftmax, cudaStream_t s);

// len[b] += cu[b+1] - cu[b], limited to cap (status recorded past it)
cudaError_t launch_cache_advance(int* len, const int* cu, int batch, long long cap, int* status, cudaStream_t s);

// ------------------------------------------------ T = 1 verification ----
cudaError_t launch_accept_sample(const float* p, const float* q, const int* draft, long long dstride,
                                 const unsigned* u, const unsigned* r, int batch, int nd, long long V, int* accept,
                                 int* next_tok, cudaStream_t s);

// --------------------------------------------------------------- KL ----
constexpr int KL_CHUNK = 8192;  // vocabulary entries per CTA of the partial-sum stage
int kl_chunks(long long V);
// partial: [rows, kl_chunks(V)] fp32 scratch
cudaError_t launch_kl_distill(const float* lt, const float* ls, long long rows, long long V, float t_kd,
                              float* kl_rows, float* kl_mean, float* partial, cudaStream_t s);
// Eq. 3 over a batch of blocks; partial: loss_partial_floats() fp32 scratch
int loss_partial_floats(int batch, int P, long long V);
cudaError_t launch_draft_loss(const float* lt, const float* ls, const int* labels, int batch, int block, int P,
                              long long V, float t_kd, float alpha, float* ce_rows, float* kl_rows, float* loss,
                              float* partial, int* status, cudaStream_t s);

// -------------------------------------------------------- attention ----
struct AttnArgs {
  const void* q;       // [M, d]  block queries (M = batch * block)
  const void* kb;      // [M, d]  block keys
  const void* vb;      // [M, d]
  const void* kc;      // [n_ctx, d] context keys
  const void* vc;      // [n_ctx, d]
  const int* cu_ctx;   // [batch + 1]; or null with ctx_len set:
  const int* ctx_len;  // [batch] cached rows: sequence b's keys are rows b * ctx_stride + [0, ctx_len[b])
  long long ctx_stride;
  int max_len;         // with ctx_len: keys past max_len are not attended (status recorded)
  void* out;           // [M, d]
  int batch, block, n_heads, head_dim, d;
  long long n_ctx;
  int chunk;           // context keys per split
  int n_chunks;        // splits per (sequence, head) = ceil(max_ctx / chunk), 1..8: one cluster
  int* status;
};
// bf16 path: TMA maps over context K/V and block K/V, box {64 cols, 64 rows}
struct AttnTmaps {
  CUtensorMap k, v, kb, vb;
};
cudaError_t launch_attention(const AttnArgs& a, const AttnTmaps* tm, int dtype, cudaStream_t s);
size_t attention_smem_bytes(int head_dim);
// clusters of `cluster` (1..8) attention CTAs resident at once; -1 if unknown
int attention_max_clusters(int head_dim, int cluster);

}  // namespace hdf
