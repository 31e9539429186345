// C ABI of libhdf (declared in include/hdf.h): host-side validation,
// workspace layout, TMA tensor-map encoding and the launch sequence of one
// block-drafting step.  Every computation runs in the CUDA kernels of this
// library; nothing here touches tensor data on the host.
#include <cudaTypedefs.h>

#include <algorithm>
#include <climits>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <atomic>
#include <map>
#include <mutex>
#include <string>
#include <tuple>
#include <utility>
#include <vector>

#include "common.cuh"
#include "kernels.h"

using namespace hdf;

// --------------------------------------------- per-device kernel set-up
namespace hdf {
namespace {
std::mutex g_setup_mu;  // guards the two tables below
// (device, kernel) -> dynamic shared-memory limit set on that device
std::map<std::pair<int, const void*>, size_t>& smem_limits() {
  static std::map<std::pair<int, const void*>, size_t> m;
  return m;
}
// (device, kernel, block, shared memory, cluster size) -> resident clusters
std::map<std::tuple<int, const void*, int, size_t, int>, int>& cluster_answers() {
  static std::map<std::tuple<int, const void*, int, size_t, int>, int> m;
  return m;
}
}  // namespace

cudaError_t ensure_smem_limit(const void* kernel, size_t smem, bool nonportable_clusters) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(g_setup_mu);
  auto& m = smem_limits();
  const auto key = std::make_pair(dev, kernel);
  const auto it = m.find(key);
  if (it != m.end() && it->second >= smem) return cudaSuccess;
  const size_t want = it == m.end() ? smem : std::max(smem, it->second);
  if ((e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)want)) != cudaSuccess)
    return e;
  if (it == m.end() && nonportable_clusters &&
      (e = cudaFuncSetAttribute(kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1)) != cudaSuccess)
    return e;
  m[key] = want;
  return cudaSuccess;
}

cudaError_t max_active_clusters(const void* kernel, int block, size_t smem, int cluster, int* n) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(g_setup_mu);
  auto& m = cluster_answers();
  const auto key = std::make_tuple(dev, kernel, block, smem, cluster);
  const auto it = m.find(key);
  if (it != m.end()) {
    *n = it->second;
    return cudaSuccess;
  }
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeClusterDimension;
  attr.val.clusterDim.x = (unsigned)cluster;
  attr.val.clusterDim.y = 1;
  attr.val.clusterDim.z = 1;
  cfg.gridDim = dim3((unsigned)cluster);
  cfg.blockDim = dim3((unsigned)block);
  cfg.dynamicSmemBytes = smem;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  int v = 0;
  if ((e = cudaOccupancyMaxActiveClusters(&v, kernel, &cfg)) != cudaSuccess) {
    cudaGetLastError();
    return e;
  }
  m[key] = v;
  *n = v;
  return cudaSuccess;
}
}  // namespace hdf

namespace {

thread_local std::string g_err;

__device__ int g_device_status;  // HDF_ERR_DEVICE_CHECK after a bounded wait ran out

int fail(int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  g_err = buf;
  return code;
}
int cuda_fail(cudaError_t e, const char* where) {
  return fail(HDF_ERR_CUDA, "%s: %s", where, cudaGetErrorString(e));
}
#define CK(call, where)                              \
  do {                                               \
    cudaError_t e_ = (call);                         \
    if (e_ != cudaSuccess) return cuda_fail(e_, where); \
  } while (0)

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
size_t esize(int dtype) { return dtype == HDF_BF16 ? 2 : 4; }
size_t up256(size_t x) { return (x + 255) & ~size_t(255); }

// Per-device caches filled on first use.  Host threads may race to fill a
// slot; they store the same value, and the slots are atomics, so the race is
// benign and defined.
int* device_status_ptr() {
  static std::atomic<int*> ptr[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
  int* p = ptr[dev].load(std::memory_order_acquire);
  if (!p) {
    void* q = nullptr;
    if (cudaGetSymbolAddress(&q, g_device_status) != cudaSuccess) return nullptr;
    p = static_cast<int*>(q);
    ptr[dev].store(p, std::memory_order_release);
  }
  return p;
}

int num_sms() {
  static std::atomic<int> cache[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
  int n = cache[dev].load(std::memory_order_relaxed);
  if (n <= 0) {
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 148;
    cache[dev].store(n, std::memory_order_relaxed);
  }
  return n;
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  // looked up once per process (the driver entry point is the same for every
  // device); the initialisation of a function-local static is thread-safe
  static const PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    return static_cast<PFN_cuTensorMapEncodeTiled_v12000>(nullptr);
  }();
  return fn;
}

// 2-D K-major map over a [rows, cols] row-major tensor (row stride ld
// elements), box {128 bytes of columns, box_rows}, 128-byte swizzle,
// zero fill outside the tensor.
int make_map(CUtensorMap* m, const void* ptr, int dtype, long long rows, long long cols, long long ld,
             int box_rows) {
  auto fn = encode_fn();
  if (!fn) return fail(HDF_ERR_CUDA, "cuTensorMapEncodeTiled unavailable");
  const size_t es = esize(dtype);
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)std::max<long long>(rows, 1)};
  cuuint64_t strides[1] = {(cuuint64_t)(ld * es)};
  cuuint32_t box[2] = {(cuuint32_t)(128 / es), (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, dtype == HDF_BF16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2,
                  const_cast<void*>(ptr), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                  CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS)
    return fail(HDF_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d) rows=%lld cols=%lld box_rows=%d", (int)r, rows,
                cols, box_rows);
  return HDF_OK;
}

// 3-D view of a bf16 H [n_tokens, m, d]: {64 elements, tokens, 128-byte
// chunks of a token row}, 128-byte swizzle, the given box.
int make_chunk_map(CUtensorMap* hm, const void* H, long long n_tokens, int m, int d, const unsigned box[3]) {
  auto fn = encode_fn();
  if (!fn) return fail(HDF_ERR_CUDA, "cuTensorMapEncodeTiled unavailable");
  cuuint64_t dims[3] = {64, (cuuint64_t)n_tokens, (cuuint64_t)((long long)m * d / 64)};
  cuuint64_t strides[2] = {(cuuint64_t)((long long)m * d * 2), 128};
  cuuint32_t bx[3] = {box[0], box[1], box[2]};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = fn(hm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(H), dims, strides, bx, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(HDF_ERR_CUDA, "cuTensorMapEncodeTiled (3-D view of H) failed (%d)", (int)r);
  return HDF_OK;
}

// ------------------------------------------------------------ GEMM plans
int pick_bn(long long n) {
  if (n <= 16) return 16;
  if (n <= 32) return 32;
  if (n <= 64) return 64;
  if (n <= 128) return 128;
  return 256;
}

struct SplitPlan {
  int bn, k_splits, tiles;
};

// Weights-as-A GEMM (rows = output features, columns = tokens), bound by
// streaming the operands through shared memory.  Two CTAs share an SM, and
// the CTAs resident at once are twice what the occupancy API gives per
// cluster size (it packs clusters into GPCs but counts one CTA per SM for a
// kernel holding tensor memory; else two per SM).  A CTA's time is about the
// bytes it loads, k-blocks x (128 + bn) rows; a split pays 2 + bn/8 k-blocks
// for storing, exchanging and summing its partial tile and waiting for the
// slowest rank of its cluster (fitted to measured plan sweeps).  The plan
// (tile width: the one covering the tokens, or 128 when that is 256; K split
// with >= 4 k-blocks per split, at most 16, one thread-block cluster per tile)
// is the one with the least waves x cost per CTA.
SplitPlan plan_swap(int dtype, long long M, long long N, long long K) {
  const int bk = dtype == HDF_BF16 ? 64 : 32;
  const int num_kb = (int)((K + bk - 1) / bk);
  const int bn0 = pick_bn(N);
  const int widths[2] = {bn0, bn0 == 256 ? 128 : 0};
  SplitPlan best{bn0, 1, (int)(((M + 127) / 128) * ((N + bn0 - 1) / bn0))};
  long long best_cost = LLONG_MAX;
  for (int bn : widths) {
    if (bn == 0) continue;
    const long long tiles = ((M + 127) / 128) * ((N + bn - 1) / bn);
    const int max_splits = bn <= 128 ? std::min(16, std::max(1, num_kb / 4)) : 1;
    for (int s = 1; s <= max_splits; ++s) {
      const int kb_per = (num_kb + s - 1) / s;
      if ((num_kb + kb_per - 1) / kb_per != s) continue;  // no empty split
      const int api = gemm_resident_ctas(dtype, bn, s);
      const long long slots = 2LL * (api > 0 ? api : num_sms());
      const long long waves = (tiles * s + slots - 1) / slots;
      const long long cost = waves * (kb_per + (s > 1 ? 2 + bn / 8 : 0)) * (128 + bn);
      if (cost < best_cost) {
        best_cost = cost;
        best = SplitPlan{bn, s, (int)tiles};
      }
    }
  }
  return best;
}

void init_gemm(GemmArgs& g, int dtype, long long M, long long N, long long K, const SplitPlan& p) {
  std::memset(&g, 0, sizeof g);
  g.M = (int)M;
  g.N = (int)N;
  g.K = (int)K;
  g.dtype = dtype;
  g.bn = p.bn;
  g.k_splits = p.k_splits;
  g.group_n = 1;
  g.status = device_status_ptr();
  g.A.rows_per_map = 1 << 30;
  g.B.rows_per_map = 1 << 30;
}

// Row-major bf16 GEMMs with 256-wide column tiles and at least 256 rows run
// on CTA pairs (gemm_pair_kernel).
bool use_pair_tiles(int dtype, int bn, long long rows) { return dtype == HDF_BF16 && bn == 256 && rows >= 256; }

// ---------------------------------------------------- draft-block layout
struct DraftLayout {
  size_t c, kc, vc, h, x, q, kb, vb, o, act, total;
  int chunk, n_chunks;
  SplitPlan qkv, oproj, gu, down;
};

// Context keys per attention CTA.  The chunks of one (sequence, head) are one
// thread-block cluster of at most 8 CTAs, each chunk at least 256 keys.  The
// count is the one with the least waves x (rounds + 2): waves of clusters
// from the resident clusters the occupancy API gives, rounds of the four
// consumer warps over the 64-key tiles of the longest chunk (the last one
// also holds the block's keys), 2 for the fixed cost of a wave; ties go to
// more chunks.
int attn_chunk(const hdf_draft_shape* sh, int* n_chunks) {
  const long long bh = std::max(1LL, (long long)sh->batch * sh->n_heads);
  const int T = sh->max_ctx;
  int best_chunk = std::max(256, ((T + 63) / 64) * 64), best_nc = 1;
  long long best_cost = LLONG_MAX;
  for (int per = 1; per <= 8; ++per) {
    const int chunk = std::max(256, (((T + per - 1) / per + 63) / 64) * 64);
    const int nc = std::max(1, (T + chunk - 1) / chunk);
    if (nc != per) continue;  // the same split as a smaller count
    const int maxc = attention_max_clusters(sh->head_dim, nc);
    const long long slots = std::max(1, maxc > 0 ? maxc : num_sms() / nc);
    const long long waves = (bh + slots - 1) / slots;
    const int last = (T - (nc - 1) * chunk + 63) / 64 + 1;
    const int tiles = std::max(chunk / 64, last);
    const long long cost = waves * ((tiles + 3) / 4 + 2);
    if (cost <= best_cost) {
      best_cost = cost;
      best_chunk = chunk;
      best_nc = nc;
    }
  }
  *n_chunks = best_nc;
  return best_chunk;
}

DraftLayout draft_layout(const hdf_draft_shape* sh) {
  DraftLayout L;
  const size_t es = esize(sh->dtype);
  const long long M = (long long)sh->batch * sh->block;
  const long long d = sh->d, F = sh->ffn;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off += up256(bytes);
    return o;
  };
  L.c = take(sh->n_ctx * d * es);
  L.kc = take(sh->n_ctx * d * es);
  L.vc = take(sh->n_ctx * d * es);
  L.h = take(M * d * 4);
  L.x = take(M * d * es);
  L.q = take(M * d * es);
  L.kb = take(M * d * es);
  L.vb = take(M * d * es);
  L.o = take(M * d * es);
  L.act = take(M * F * es);
  L.chunk = attn_chunk(sh, &L.n_chunks);
  // The block path's Q / K_b / V_b projection runs beside the context
  // projection (cold step) or the append (serving round), on the SM slots
  // those leave: it takes no K split, which would multiply its CTAs past those
  // slots and queue them behind the projection.
  L.qkv = plan_swap(sh->dtype, 3 * d, M, d);
  L.qkv.k_splits = 1;
  L.oproj = plan_swap(sh->dtype, d, M, d);
  L.gu = plan_swap(sh->dtype, 2 * F, M, d);
  L.down = plan_swap(sh->dtype, d, M, F);
  L.total = off;
  return L;
}

int check_draft_shape(const hdf_draft_shape* sh) {
  if (!sh) return fail(HDF_ERR_INVALID_ARG, "shape is NULL");
  if (sh->dtype != HDF_BF16 && sh->dtype != HDF_F32) return fail(HDF_ERR_DTYPE, "dtype %d", sh->dtype);
  if (sh->batch < 0 || sh->block < 2 || sh->block > 16)
    return fail(HDF_ERR_SHAPE, "batch %d / block %d (need block in 2..16)", sh->batch, sh->block);
  if (sh->d <= 0 || sh->d % 128) return fail(HDF_ERR_SHAPE, "d=%d must be a positive multiple of 128", sh->d);
  if (sh->head_dim != 64 && sh->head_dim != 128) return fail(HDF_ERR_SHAPE, "head_dim %d", sh->head_dim);
  if ((long long)sh->n_heads * sh->head_dim != sh->d) return fail(HDF_ERR_SHAPE, "n_heads*head_dim != d");
  if (sh->ffn <= 0 || sh->ffn % 64) return fail(HDF_ERR_SHAPE, "ffn=%d must be a multiple of 64", sh->ffn);
  if (sh->vocab <= 0 || sh->n_layers < 1) return fail(HDF_ERR_SHAPE, "vocab/n_layers");
  if (sh->n_ctx < 0 || sh->max_ctx < 0 || sh->n_ctx > 0x7fffffffLL)
    return fail(HDF_ERR_SHAPE, "n_ctx/max_ctx");
  if ((long long)sh->batch * sh->block > 4096) return fail(HDF_ERR_UNSUPPORTED, "batch*block > 4096");
  if (!(sh->norm_eps >= 0.f)) return fail(HDF_ERR_INVALID_ARG, "norm_eps");
  return HDF_OK;
}

}  // namespace

// =====================================================================
extern "C" {

int hdf_version(void) { return 102; }

const char* hdf_status_str(int s) {
  switch (s) {
    case HDF_OK: return "ok";
    case HDF_ERR_INVALID_ARG: return "invalid argument";
    case HDF_ERR_SHAPE: return "unsupported or inconsistent shape";
    case HDF_ERR_DTYPE: return "unknown dtype";
    case HDF_ERR_ALIGNMENT: return "pointer not 16-byte aligned";
    case HDF_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
    case HDF_ERR_CUDA: return "CUDA error";
    case HDF_ERR_UNSUPPORTED: return "unsupported configuration";
    case HDF_ERR_DEVICE_CHECK: return "device-side bounded wait expired";
    default: return "unknown status";
  }
}

const char* hdf_last_error(void) { return g_err.c_str(); }

int hdf_device_status(int reset) {
  CK(cudaDeviceSynchronize(), "cudaDeviceSynchronize");
  int v = 0;
  CK(cudaMemcpyFromSymbol(&v, g_device_status, sizeof v), "cudaMemcpyFromSymbol");
  if (reset) {
    const int z = 0;
    CK(cudaMemcpyToSymbol(g_device_status, &z, sizeof z), "cudaMemcpyToSymbol");
  }
  return v;
}

// ---------------------------------------------------- reducer backward
namespace {
struct ReduceBwdLayout {
  size_t u, dg, part, dbpart, total;
};
ReduceBwdLayout reduce_bwd_layout(const ReduceBwdPlan& p, long long n, int m, int d) {
  ReduceBwdLayout L;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off += up256(bytes);
    return o;
  };
  L.u = take((size_t)n * m * 4);
  L.dg = take((size_t)n * m * 4);
  L.part = take((size_t)p.splits * m * m * d * 4);
  L.dbpart = take((size_t)p.splits * m * 4);
  L.total = n > 0 ? off : 0;
  return L;
}
int check_reduce_bwd(int dtype, int64_t n_tokens, int m, int d) {
  if (dtype != HDF_BF16 && dtype != HDF_F32) return fail(HDF_ERR_DTYPE, "dtype %d", dtype);
  if (n_tokens < 0) return fail(HDF_ERR_SHAPE, "n_tokens < 0");
  if (!(m == 1 || m == 2 || m == 3 || m == 4 || m == 8)) return fail(HDF_ERR_UNSUPPORTED, "m=%d", m);
  const int vec = dtype == HDF_BF16 ? 8 : 4;
  if (d <= 0 || d % vec || d > 16384) return fail(HDF_ERR_SHAPE, "d=%d (multiple of %d, <= 16384)", d, vec);
  return HDF_OK;
}
}  // namespace

size_t hdf_gated_reduce_backward_workspace_size(int64_t n_tokens, int m, int d, int dtype) {
  if (check_reduce_bwd(dtype, n_tokens, m, d)) return 0;
  return reduce_bwd_layout(reduce_bwd_plan(n_tokens, m, d, dtype, num_sms()), n_tokens, m, d).total;
}

int hdf_gated_reduce_backward(const void* H, int dtype, int64_t n_tokens, int m, int d, const void* Wf,
                              const float* b, float rms_eps, float gate_scale, const void* dy, float* dWf,
                              float* db, void* ws, size_t ws_bytes, hdf_stream_t stream) {
  g_err.clear();
  int rc;
  if ((rc = check_reduce_bwd(dtype, n_tokens, m, d))) return rc;
  if (!dWf || !db) return fail(HDF_ERR_INVALID_ARG, "dWf and db are required");
  if (!aligned16(dWf)) return fail(HDF_ERR_ALIGNMENT, "dWf must be 16-byte aligned");
  const cudaStream_t s = (cudaStream_t)stream;
  if (n_tokens == 0) {  // empty sums
    CK(cudaMemsetAsync(dWf, 0, (size_t)m * m * d * 4, s), "memset dWf");
    CK(cudaMemsetAsync(db, 0, (size_t)m * 4, s), "memset db");
    return HDF_OK;
  }
  if (!H || !Wf || !b || !dy) return fail(HDF_ERR_INVALID_ARG, "H, Wf, b and dy are required");
  if (!aligned16(H) || !aligned16(Wf) || !aligned16(dy))
    return fail(HDF_ERR_ALIGNMENT, "H, Wf and dy must be 16-byte aligned");
  if (!std::isfinite(rms_eps) || !std::isfinite(gate_scale) || rms_eps < 0)
    return fail(HDF_ERR_INVALID_ARG, "non-finite or negative scalar");
  const ReduceBwdPlan p = reduce_bwd_plan(n_tokens, m, d, dtype, num_sms());
  const ReduceBwdLayout L = reduce_bwd_layout(p, n_tokens, m, d);
  if (!ws || ws_bytes < L.total || (reinterpret_cast<uintptr_t>(ws) & 255))
    return fail(HDF_ERR_WORKSPACE, "workspace %zu bytes (need %zu, 256-byte aligned)", ws_bytes, L.total);
  char* W = static_cast<char*>(ws);
  ReduceBwdArgs a;
  a.H = H;
  a.Wf = Wf;
  a.b = b;
  a.dy = dy;
  a.dWf = dWf;
  a.db = db;
  a.u = reinterpret_cast<float*>(W + L.u);
  a.dg = reinterpret_cast<float*>(W + L.dg);
  a.part = reinterpret_cast<float*>(W + L.part);
  a.dbpart = reinterpret_cast<float*>(W + L.dbpart);
  a.n_tokens = n_tokens;
  a.m = m;
  a.d = d;
  a.rms_eps = rms_eps;
  a.gate_scale = gate_scale;
  CK(launch_gated_reduce_backward(a, dtype, p, s), "gated_reduce backward launch");
  return HDF_OK;
}

// ------------------------------------------------------------- reducer
int hdf_gated_reduce(const void* H, int dtype, int64_t n_tokens, int m, int d, const void* Wf, const float* b,
                     float rms_eps, float gate_scale, float gate_offset, const void* path_norm_w,
                     float path_norm_eps, const float* alpha_override, void* y, float* alpha_out,
                     hdf_stream_t stream) {
  return hdf_gated_reduce_kernel(HDF_REDUCE_AUTO, H, dtype, n_tokens, m, d, Wf, b, rms_eps, gate_scale, gate_offset,
                                 path_norm_w, path_norm_eps, alpha_override, y, alpha_out, stream);
}

int hdf_gated_reduce_kernel(int path, const void* H, int dtype, int64_t n_tokens, int m, int d, const void* Wf,
                            const float* b, float rms_eps, float gate_scale, float gate_offset,
                            const void* path_norm_w, float path_norm_eps, const float* alpha_override, void* y,
                            float* alpha_out, hdf_stream_t stream) {
  g_err.clear();
  if (path != HDF_REDUCE_AUTO && path != HDF_REDUCE_GENERAL && path != HDF_REDUCE_CLUSTER && path != HDF_REDUCE_TILE)
    return fail(HDF_ERR_INVALID_ARG, "reduce kernel %d", path);
  if (dtype != HDF_BF16 && dtype != HDF_F32) return fail(HDF_ERR_DTYPE, "dtype %d", dtype);
  if (n_tokens < 0) return fail(HDF_ERR_SHAPE, "n_tokens < 0");
  if (!(m == 1 || m == 2 || m == 3 || m == 4 || m == 8)) return fail(HDF_ERR_UNSUPPORTED, "m=%d", m);
  const int vec = dtype == HDF_BF16 ? 8 : 4;
  if (d <= 0 || d % vec || d > 16384) return fail(HDF_ERR_SHAPE, "d=%d (multiple of %d, <= 16384)", d, vec);
  if (n_tokens == 0) return HDF_OK;
  if (!H || !y) return fail(HDF_ERR_INVALID_ARG, "H and y are required");
  if (!alpha_override && (!Wf || !b)) return fail(HDF_ERR_INVALID_ARG, "Wf and b are required without override");
  if (!aligned16(H) || !aligned16(y) || (Wf && !aligned16(Wf)) || (path_norm_w && !aligned16(path_norm_w)))
    return fail(HDF_ERR_ALIGNMENT, "H, Wf, path_norm_w and y must be 16-byte aligned");
  if (!std::isfinite(rms_eps) || !std::isfinite(gate_scale) || !std::isfinite(gate_offset) ||
      !std::isfinite(path_norm_eps) || rms_eps < 0 || path_norm_eps < 0)
    return fail(HDF_ERR_INVALID_ARG, "non-finite or negative scalar");
  int rc;
  ReduceArgs a;
  a.H = H;
  a.Wf = Wf;
  a.b = b;
  a.path_norm_w = path_norm_w;
  a.alpha_override = alpha_override;
  a.y = y;
  a.alpha_out = alpha_out;
  a.n_tokens = n_tokens;
  a.m = m;
  a.d = d;
  a.rms_eps = rms_eps;
  a.gate_scale = gate_scale;
  a.gate_offset = gate_offset;
  a.path_norm_eps = path_norm_eps;
  a.status = device_status_ptr();
  unsigned box[3];
  unsigned tail_box[3];
  // auto: the tile kernel for m = 4 (1.2-1.6x the general kernel from 4096
  // tokens, a tie below), the general kernel for other m.  The choice does not
  // depend on n_tokens: a token's y is then the same bits whether it is
  // reduced with its whole context or alone in a serving round.
  const bool tile_wanted = path == HDF_REDUCE_TILE || (path == HDF_REDUCE_AUTO && m == 4);
  if (tile_wanted && reduce_tile_boxes(a, dtype, box, tail_box)) {
    CUtensorMap hm[2];
    if ((rc = make_chunk_map(&hm[0], H, n_tokens, m, d, box))) return rc;
    if ((rc = make_chunk_map(&hm[1], H, n_tokens, m, d, tail_box))) return rc;
    CK(launch_gated_reduce_tile(a, hm, (cudaStream_t)stream), "gated_reduce tile launch");
    return HDF_OK;
  }
  const bool cluster_wanted = path == HDF_REDUCE_CLUSTER;
  if (cluster_wanted && reduce_cluster_box(a, dtype, box)) {
    CUtensorMap hm;
    if ((rc = make_chunk_map(&hm, H, n_tokens, m, d, box))) return rc;
    CK(launch_gated_reduce_cluster(a, &hm, (cudaStream_t)stream), "gated_reduce cluster launch");
    return HDF_OK;
  }
  CK(launch_gated_reduce(a, dtype, (cudaStream_t)stream), "gated_reduce launch");
  return HDF_OK;
}

// -------------------------------------------------------- fc comparison
size_t hdf_fc_reduce_workspace_size(int64_t, int, int, int, int) { return 0; }

int hdf_fc_reduce(const void* H, int dtype, int64_t n_tokens, int m, int d_in, int d_out, const void* W_fc, void* y,
                  void*, size_t, hdf_stream_t stream) {
  g_err.clear();
  if (dtype != HDF_BF16 && dtype != HDF_F32) return fail(HDF_ERR_DTYPE, "dtype %d", dtype);
  if (n_tokens < 0 || m < 1 || d_in <= 0 || d_out <= 0 || d_out % 128)
    return fail(HDF_ERR_SHAPE, "need m >= 1, d_in > 0 and d_out %% 128 == 0 (m %d, d_in %d, d_out %d)", m, d_in,
                d_out);
  if ((long long)m * d_in * esize(dtype) % 16) return fail(HDF_ERR_SHAPE, "row stride m * d_in not 16-byte aligned");
  if (n_tokens == 0) return HDF_OK;
  if (!H || !W_fc || !y) return fail(HDF_ERR_INVALID_ARG, "null pointer");
  if (!aligned16(H) || !aligned16(W_fc) || !aligned16(y)) return fail(HDF_ERR_ALIGNMENT, "alignment");
  if (n_tokens > 0x7fffffffLL) return fail(HDF_ERR_SHAPE, "n_tokens too large");
  const long long K = (long long)m * d_in;
  SplitPlan p{d_out % 256 == 0 ? 256 : 128, 1, 0};
  GemmArgs g;
  init_gemm(g, dtype, n_tokens, d_out, K, p);
  g.group_n = 8;
  g.pair = use_pair_tiles(dtype, p.bn, n_tokens);
  int rc;
  if ((rc = make_map(&g.A.map[0], H, dtype, n_tokens, K, K, 64))) return rc;
  if ((rc = make_map(&g.B.map[0], W_fc, dtype, d_out, K, K, g.pair ? 128 : p.bn))) return rc;
  g.pre_operand = 2;  // the weight
  g.epi.kind = kEpiStore;
  g.epi.out[0] = y;
  g.epi.seg_width = d_out;
  g.epi.ld = d_out;
  if (g.pair) {
    if ((rc = make_map(&g.epi.out_map[0], y, dtype, n_tokens, d_out, d_out, 128))) return rc;
    g.epi.out_tma = 1;
  }
  CK(launch_gemm(g, (cudaStream_t)stream), "fc gemm launch");
  return HDF_OK;
}

// --------------------------------------------------------------- RoPE
int hdf_rope_table(double theta, int head_dim, int64_t max_pos, float* cos_out, float* sin_out,
                   hdf_stream_t stream) {
  g_err.clear();
  if (!(theta > 0) || head_dim <= 0 || head_dim % 2 || max_pos < 0)
    return fail(HDF_ERR_INVALID_ARG, "theta/head_dim/max_pos");
  if (max_pos == 0) return HDF_OK;
  if (!cos_out || !sin_out) return fail(HDF_ERR_INVALID_ARG, "null output");
  CK(launch_rope_table(theta, head_dim, max_pos, cos_out, sin_out, (cudaStream_t)stream), "rope launch");
  return HDF_OK;
}

// --------------------------------------------------------- draft block
}  // extern "C"

namespace {

// Weight pointers and RoPE table of a draft call: non-null and 16-byte aligned.
int check_drafter_weights(const hdf_drafter_weights* w, const hdf_draft_shape* sh) {
  if (!w || !w->layers) return fail(HDF_ERR_INVALID_ARG, "weights / layers NULL");
  if (!w->embed || !w->mask_vec || !w->ctx_norm || !w->final_norm || !w->rope_cos || !w->rope_sin)
    return fail(HDF_ERR_INVALID_ARG, "null weight");
  const void* ptrs[] = {w->embed, w->mask_vec, w->ctx_norm, w->final_norm};
  for (const void* p : ptrs)
    if (!aligned16(p)) return fail(HDF_ERR_ALIGNMENT, "weight not 16-byte aligned");
  for (int l = 0; l < sh->n_layers; ++l) {
    const hdf_layer_weights& L = w->layers[l];
    const void* lp[] = {L.attn_norm, L.wq, L.wk, L.wv, L.wo, L.mlp_norm, L.wg, L.wu, L.wd};
    for (const void* p : lp) {
      if (!p) return fail(HDF_ERR_INVALID_ARG, "layer %d weight NULL", l);
      if (!aligned16(p)) return fail(HDF_ERR_ALIGNMENT, "layer %d weight misaligned", l);
    }
  }
  return HDF_OK;
}

int check_cache(const hdf_ctx_cache* cache, const hdf_draft_shape* sh) {
  if (!cache || !cache->k || !cache->v || !cache->len) return fail(HDF_ERR_INVALID_ARG, "cache / k / v / len NULL");
  if (!aligned16(cache->k) || !aligned16(cache->v) || (reinterpret_cast<uintptr_t>(cache->len) & 3))
    return fail(HDF_ERR_ALIGNMENT, "cache k / v must be 16-byte aligned, len 4-byte aligned");
  if (cache->capacity < 1) return fail(HDF_ERR_SHAPE, "cache capacity %d", cache->capacity);
  if ((long long)sh->batch * cache->capacity > 0x7fffffffLL)
    return fail(HDF_ERR_SHAPE, "batch * capacity must stay below 2^31 rows");
  return HDF_OK;
}

// Byte offset of layer l in a cache tensor [n_layers, batch, capacity, d].
size_t cache_layer_offset(const hdf_draft_shape* sh, const hdf_ctx_cache* cache, int l) {
  return (size_t)l * sh->batch * (size_t)cache->capacity * sh->d * esize(sh->dtype);
}

// Context rows up to which the K/V projection runs weights-as-A: the
// weight rows fill the 128-row tiles and the few context rows ride in one
// narrow column tile, instead of a 128-row tile of mostly absent rows that
// every CTA of the grid reads at once.
constexpr long long kCtxKvSwapRows = 256;

// Tile width of the row-major context K/V GEMM: 256 columns when a 256-wide
// grid covers every SM (the projection of a whole context is compute-bound);
// otherwise the widest tile that still gives two CTAs per SM, down to 16.
int ctx_kv_bn(const hdf_draft_shape* sh, long long rows) {
  const long long row_tiles = (rows + 127) / 128;
  if (sh->d % 256 == 0 && row_tiles * (2LL * sh->d / 256) >= num_sms()) return 256;
  int bn = 128;
  while (bn > 16 && row_tiles * (2LL * sh->d / bn) < 2LL * num_sms()) bn >>= 1;
  return bn;
}

// [K_c | V_c] = c [W_k; W_v]^T with RoPE on K_c.  Never a K split: each
// output element is one K-ordered accumulation whatever the orientation or
// tile width, so a row's K / V do not depend on the launch that made them.
// pos_mode 1: rows land packed in kout / vout; pos_mode 3: rows are appended
// to a cache (cu = cu_new, len, cap).
int launch_ctx_kv(const hdf_drafter_weights* w, const hdf_layer_weights& Lw, const hdf_draft_shape* sh,
                  const void* c, long long rows, void* kout, void* vout, const int32_t* cu, int pos_mode,
                  const int32_t* len, long long cap, cudaStream_t s) {
  const int dt = sh->dtype;
  const long long d = sh->d;
  const bool swap = rows <= kCtxKvSwapRows;
  GemmArgs g;
  int rc;
  if (swap) {  // rows = output features of [W_k; W_v], columns = context rows
    const SplitPlan p{pick_bn(rows), 1, 0};
    init_gemm(g, dt, 2 * d, rows, d, p);
    if ((rc = make_map(&g.A.map[0], Lw.wk, dt, d, d, d, 64))) return rc;
    if ((rc = make_map(&g.A.map[1], Lw.wv, dt, d, d, d, 64))) return rc;
    g.A.rows_per_map = (int)d;
    if ((rc = make_map(&g.B.map[0], c, dt, rows, d, d, p.bn))) return rc;
    g.pre_operand = 1;  // weights: loaded before the context norm has finished
    g.epi.kind = kEpiStoreT;
  } else {
    const SplitPlan p{ctx_kv_bn(sh, rows), 1, 0};
    init_gemm(g, dt, rows, 2 * d, d, p);
    g.group_n = 8;
    // 256-wide tiles run as 256 x 256 tiles on CTA pairs: each CTA loads
    // 128 rows of the weights
    g.pair = use_pair_tiles(dt, p.bn, rows);
    const int b_box = g.pair ? 128 : p.bn;
    if ((rc = make_map(&g.A.map[0], c, dt, rows, d, d, 64))) return rc;
    if ((rc = make_map(&g.B.map[0], Lw.wk, dt, d, d, d, b_box))) return rc;
    if ((rc = make_map(&g.B.map[1], Lw.wv, dt, d, d, d, b_box))) return rc;
    g.pre_operand = 2;
    g.B.rows_per_map = (int)d;
    g.epi.kind = kEpiStore;
  }
  g.epi.out[0] = kout;
  g.epi.out[1] = vout;
  g.epi.seg_width = (int)d;
  g.epi.ld = d;
  g.epi.rope_mask = 1;
  g.epi.rope_cos = w->rope_cos;
  g.epi.rope_sin = w->rope_sin;
  g.epi.rope_rows = w->rope_max_pos;
  g.epi.head_dim = sh->head_dim;
  g.epi.cu_ctx = cu;
  g.epi.batch = sh->batch;
  g.epi.block = sh->block;
  g.epi.pos_mode = pos_mode;
  g.epi.ctx_len = len;
  g.epi.cache_cap = cap;
  if (g.pair && pos_mode == 1) {  // packed rows: the tile leaves by TMA stores
    if ((rc = make_map(&g.epi.out_map[0], kout, dt, rows, d, d, 128))) return rc;
    if ((rc = make_map(&g.epi.out_map[1], vout, dt, rows, d, d, 128))) return rc;
    g.epi.out_tma = 1;
  }
  CK(launch_gemm(g, s), "ctx kv gemm");
  return HDF_OK;
}

// Second stream of the calling thread on the current device, with events
// for fork / join points.  Created once, in relaxed capture mode so that a
// first call made under stream capture may create it.  nullptr on failure.
struct SideStream {
  cudaStream_t s = nullptr;
  std::vector<cudaEvent_t> ev;
};
SideStream* side_stream(size_t n_events) {
  thread_local SideStream per_dev[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
  SideStream& ss = per_dev[dev];
  if (ss.s && ss.ev.size() >= n_events) return &ss;
  cudaStreamCaptureMode mode = cudaStreamCaptureModeRelaxed;
  cudaThreadExchangeStreamCaptureMode(&mode);
  bool ok = true;
  if (!ss.s) {
    // the context path (norm, then each layer's K/V projection) is the
    // step's critical path: its CTAs go first when both streams have work
    int least = 0, greatest = 0;
    if (cudaDeviceGetStreamPriorityRange(&least, &greatest) != cudaSuccess) greatest = 0;
    ok = cudaStreamCreateWithPriority(&ss.s, cudaStreamNonBlocking, greatest) == cudaSuccess;
  }
  while (ok && ss.ev.size() < n_events) {
    cudaEvent_t e;
    ok = cudaEventCreateWithFlags(&e, cudaEventDisableTiming) == cudaSuccess;
    if (ok) ss.ev.push_back(e);
  }
  cudaThreadExchangeStreamCaptureMode(&mode);
  if (!ok) {
    if (ss.s) cudaStreamDestroy(ss.s);
    ss.s = nullptr;
    return nullptr;
  }
  return &ss;
}

// New context rows of a serving round (hdf_draft_round): their reduced
// states, row offsets, count and the workspace their normed copy goes to.
struct AppendIn {
  const void* ctx_new;
  const int32_t* cu_new;
  long long n_new;
  void* c;
};

// c = RMSNorm(ctx_new), then every layer's K_c / V_c rows written at
// positions len[i].. of the cache (mode 3); the lengths are left alone.
int append_rows(const hdf_drafter_weights* w, const hdf_draft_shape* sh, const AppendIn& ap,
                const hdf_ctx_cache* cache, cudaStream_t s) {
  int rc;
  CK(launch_rmsnorm(ap.ctx_new, 0, w->ctx_norm, ap.c, sh->dtype, ap.n_new, sh->d, sh->norm_eps, s), "ctx norm");
  for (int l = 0; l < sh->n_layers; ++l) {
    char* kl = static_cast<char*>(cache->k) + cache_layer_offset(sh, cache, l);
    char* vl = static_cast<char*>(cache->v) + cache_layer_offset(sh, cache, l);
    if ((rc = launch_ctx_kv(w, w->layers[l], sh, ap.c, ap.n_new, kl, vl, ap.cu_new, 3, cache->len,
                            cache->capacity, s)))
      return rc;
  }
  return HDF_OK;
}

// The block forward of hdf_draft_block.  Context from packed rows (ctx,
// cu_ctx: normed and projected here) or from a K/V cache (cache != null).
// With ap (cached only): the serving round, new rows appended first.
int draft_forward(const hdf_drafter_weights* w, const hdf_draft_shape* sh, const void* ctx, const int32_t* cu_ctx,
                  const hdf_ctx_cache* cache, const int32_t* anchor, void* h_out, void* ws, size_t ws_bytes,
                  const hdf_trace* trace, cudaStream_t s, const AppendIn* ap = nullptr) {
  int rc;
  const int dt = sh->dtype;
  const long long M = (long long)sh->batch * sh->block;
  const long long d = sh->d, F = sh->ffn;
  const bool cached = cache != nullptr;
  hdf_draft_shape lsh = *sh;
  if (cached) lsh.n_ctx = 0;  // no context rows to project: the layout holds the block only
  const DraftLayout Lo = draft_layout(&lsh);
  if (!ws || ws_bytes < Lo.total || (reinterpret_cast<uintptr_t>(ws) & 255))
    return fail(HDF_ERR_WORKSPACE, "workspace %zu bytes (need %zu, 256-byte aligned)", ws_bytes, Lo.total);
  char* W = static_cast<char*>(ws);
  void* c = W + Lo.c;
  void* kc = W + Lo.kc;
  void* vc = W + Lo.vc;
  float* h = reinterpret_cast<float*>(W + Lo.h);
  void* x = W + Lo.x;
  void* q = W + Lo.q;
  void* kbk = W + Lo.kb;
  void* vbk = W + Lo.vb;
  void* o = W + Lo.o;
  void* act = W + Lo.act;
  const long long n_ctx = cached ? 0 : sh->n_ctx;

  const int n_ev = trace ? trace->n_events : 0;
  const int want_ev = 3 + HDF_DRAFT_STAGES_PER_LAYER * sh->n_layers;
  if (trace && (!trace->events || n_ev != want_ev)) return fail(HDF_ERR_INVALID_ARG, "trace needs %d events", want_ev);
  int ev_i = 0;
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  if (trace) CK(cudaStreamIsCapturing(s, &cap), "cudaStreamIsCapturing");
  // under stream capture the records become external event nodes of the
  // graph, so the stage times stay measurable when the graph is replayed
  auto mark = [&]() -> int {
    if (!trace) return HDF_OK;
    cudaEvent_t ev = (cudaEvent_t)trace->events[ev_i++];
    if (cap == cudaStreamCaptureStatusActive)
      CK(cudaEventRecordWithFlags(ev, s, cudaEventRecordExternal), "cudaEventRecordWithFlags");
    else
      CK(cudaEventRecord(ev, s), "cudaEventRecord");
    return HDF_OK;
  };

  // Each layer's context K/V projection (compute-bound) and its block path
  // (input norm and Q/K_b/V_b projection: weight streaming) run on two
  // streams and join before the layer's attention.  Layer 0's projection
  // is the step's critical path (behind the reduce and the context norm): it
  // stays on the caller's stream and the block path is forked onto a second
  // stream only after the context norm, so that the projection's CTAs take
  // the SMs first and the few CTAs of the block path fill the rest.  Later
  // layers' projections go on the second stream, forked once the previous
  // layer's attention has read the shared K/V buffers, beside that layer's
  // MLP and the next block path.  Serial when stage times are traced.
  //
  // In a serving round the new rows' append (norm and every layer's K/V
  // rows) stays on the caller's stream and the first block path is forked
  // before it; the lengths advance after both, before the first attention.
  const bool round = cached && ap && ap->n_new > 0;
  SideStream* side = nullptr;
  if (!trace && (n_ctx > 0 || round)) side = side_stream(2 * (size_t)sh->n_layers + 1);
  const cudaStream_t s2 = side ? side->s : s;
  const bool beside_append = round && side;
  if (round) {
    if (side) CK(cudaEventRecord(side->ev[0], s), "fork record");  // the block path needs nothing new
    if ((rc = append_rows(w, sh, *ap, cache, s))) return rc;
    if (!side)
      CK(launch_cache_advance(cache->len, ap->cu_new, sh->batch, cache->capacity, device_status_ptr(), s),
         "cache advance");
  }
  // ---- context RMSNorm
  if ((rc = mark())) return rc;
  if (n_ctx > 0) CK(launch_rmsnorm(ctx, 0, w->ctx_norm, c, dt, n_ctx, (int)d, sh->norm_eps, s), "ctx norm");

  for (int l = 0; l < sh->n_layers; ++l) {
    const hdf_layer_weights& Lw = w->layers[l];
    // streams of this layer's projection and block path
    const cudaStream_t s_ctx = l == 0 ? s : s2;
    const cudaStream_t s_blk = l == 0 ? s2 : s;
    // ---- conditioning projection: [K_c | V_c] = c [W_k; W_v]^T, RoPE on K_c
    if ((rc = mark())) return rc;
    if (side && l == 0 && !round) CK(cudaEventRecord(side->ev[0], s), "fork record");  // behind the context norm
    if (side && l > 0) CK(cudaStreamWaitEvent(s2, side->ev[2 * l], 0), "fork wait");  // behind attention l-1
    if (n_ctx > 0 &&
        (rc = launch_ctx_kv(w, Lw, sh, c, n_ctx, kc, vc, cu_ctx, 1, nullptr, 0, s_ctx)))
      return rc;
    if (side && l == 0) CK(cudaStreamWaitEvent(s2, side->ev[0], 0), "fork wait");
    if (side && l > 0) CK(cudaEventRecord(side->ev[2 * l + 1], s2), "join record");
    // context K / V of this layer: the workspace, or the cache
    const void* kctx = kc;
    const void* vctx = vc;
    long long ctx_rows = n_ctx;
    if (cached) {
      kctx = static_cast<const char*>(cache->k) + cache_layer_offset(sh, cache, l);
      vctx = static_cast<const char*>(cache->v) + cache_layer_offset(sh, cache, l);
      ctx_rows = (long long)sh->batch * cache->capacity;
    }
    // ---- block input / attention norm
    if ((rc = mark())) return rc;
    if (l == 0)
      CK(launch_embed_norm(w->embed, w->mask_vec, anchor, Lw.attn_norm, h, x, dt, sh->batch, sh->block, (int)d,
                           sh->vocab, sh->norm_eps, s_blk),
         "embed norm");
    else
      CK(launch_rmsnorm(h, 1, Lw.attn_norm, x, dt, M, (int)d, sh->norm_eps, s_blk), "attn norm");
    // ---- Q / K_b / V_b with RoPE at block positions
    if ((rc = mark())) return rc;
    {
      GemmArgs g;
      init_gemm(g, dt, 3 * d, M, d, Lo.qkv);
      if ((rc = make_map(&g.A.map[0], Lw.wq, dt, d, d, d, 64))) return rc;
      if ((rc = make_map(&g.A.map[1], Lw.wk, dt, d, d, d, 64))) return rc;
      if ((rc = make_map(&g.A.map[2], Lw.wv, dt, d, d, d, 64))) return rc;
      g.A.rows_per_map = (int)d;
      if ((rc = make_map(&g.B.map[0], x, dt, M, d, d, Lo.qkv.bn))) return rc;
      g.pre_operand = 1;
      g.epi.kind = kEpiStoreT;
      g.epi.out[0] = q;
      g.epi.out[1] = kbk;
      g.epi.out[2] = vbk;
      g.epi.seg_width = (int)d;
      g.epi.ld = d;
      g.epi.rope_mask = 3;
      g.epi.rope_cos = w->rope_cos;
      g.epi.rope_sin = w->rope_sin;
      g.epi.rope_rows = w->rope_max_pos;
      g.epi.head_dim = sh->head_dim;
      const bool pending = beside_append && l == 0;  // the lengths do not count the new rows yet
      g.epi.cu_ctx = pending ? ap->cu_new : cu_ctx;
      g.epi.ctx_len = cached ? cache->len : nullptr;
      g.epi.batch = sh->batch;
      g.epi.block = sh->block;
      g.epi.pos_mode = cached ? (pending ? 5 : 4) : 2;
      CK(launch_gemm(g, s_blk), "qkv gemm");
      if (side && l == 0) CK(cudaEventRecord(side->ev[1], s2), "join record");
    }
    // ---- attention over [K_c; K_b]
    if ((rc = mark())) return rc;
    {
      AttnArgs a;
      std::memset(&a, 0, sizeof a);
      a.q = q;
      a.kb = kbk;
      a.vb = vbk;
      a.kc = kctx;
      a.vc = vctx;
      a.cu_ctx = cached ? nullptr : cu_ctx;
      a.ctx_len = cached ? cache->len : nullptr;
      a.ctx_stride = cached ? cache->capacity : 0;
      a.max_len = sh->max_ctx;
      a.out = o;
      a.batch = sh->batch;
      a.block = sh->block;
      a.n_heads = sh->n_heads;
      a.head_dim = sh->head_dim;
      a.d = (int)d;
      a.n_ctx = ctx_rows;
      a.chunk = Lo.chunk;
      a.n_chunks = Lo.n_chunks;
      a.status = device_status_ptr();
      AttnTmaps tm;
      if (dt == HDF_BF16) {
        const void* kc_src = ctx_rows > 0 ? kctx : kbk;
        const void* vc_src = ctx_rows > 0 ? vctx : vbk;
        const long long rows = ctx_rows > 0 ? ctx_rows : M;
        if ((rc = make_map(&tm.k, kc_src, dt, rows, d, d, 64))) return rc;
        if ((rc = make_map(&tm.v, vc_src, dt, rows, d, d, 64))) return rc;
        if ((rc = make_map(&tm.kb, kbk, dt, M, d, d, 64))) return rc;
        if ((rc = make_map(&tm.vb, vbk, dt, M, d, d, 64))) return rc;
      }
      if (side) CK(cudaStreamWaitEvent(s, side->ev[2 * l + 1], 0), "join wait");
      if (beside_append && l == 0)
        CK(launch_cache_advance(cache->len, ap->cu_new, sh->batch, cache->capacity, device_status_ptr(), s),
           "cache advance");
      CK(launch_attention(a, &tm, dt, s), "attention");
      if (side && l + 1 < sh->n_layers) CK(cudaEventRecord(side->ev[2 * l + 2], s), "attention-done record");
    }
    // ---- h += O W_o^T
    if ((rc = mark())) return rc;
    {
      GemmArgs g;
      init_gemm(g, dt, d, M, d, Lo.oproj);
      if ((rc = make_map(&g.A.map[0], Lw.wo, dt, d, d, d, 64))) return rc;
      if ((rc = make_map(&g.B.map[0], o, dt, M, d, d, Lo.oproj.bn))) return rc;
      g.pre_operand = 1;
      g.epi.kind = kEpiResidT;
      g.epi.resid = h;
      g.epi.ld = d;
      CK(launch_gemm(g, s), "o gemm");
    }
    // ---- MLP norm
    if ((rc = mark())) return rc;
    CK(launch_rmsnorm(h, 1, Lw.mlp_norm, x, dt, M, (int)d, sh->norm_eps, s), "mlp norm");
    // ---- act = silu(x W_g^T) * (x W_u^T)
    if ((rc = mark())) return rc;
    {
      GemmArgs g;
      init_gemm(g, dt, 2 * F, M, d, Lo.gu);
      if ((rc = make_map(&g.A.map[0], Lw.wg, dt, F, d, d, 64))) return rc;
      if ((rc = make_map(&g.A.map[1], Lw.wu, dt, F, d, d, 64))) return rc;
      g.A.mode = kPair64;
      if ((rc = make_map(&g.B.map[0], x, dt, M, d, d, Lo.gu.bn))) return rc;
      g.pre_operand = 1;
      g.epi.kind = kEpiSwigluT;
      g.epi.out[0] = act;
      g.epi.seg_width = (int)F;
      g.epi.ld = F;
      CK(launch_gemm(g, s), "gate/up gemm");
    }
    // ---- h += act W_d^T
    if ((rc = mark())) return rc;
    {
      GemmArgs g;
      init_gemm(g, dt, d, M, F, Lo.down);
      if ((rc = make_map(&g.A.map[0], Lw.wd, dt, d, F, F, 64))) return rc;
      if ((rc = make_map(&g.B.map[0], act, dt, M, F, F, Lo.down.bn))) return rc;
      g.pre_operand = 1;
      g.epi.kind = kEpiResidT;
      g.epi.resid = h;
      g.epi.ld = d;
      CK(launch_gemm(g, s), "down gemm");
    }
  }
  // ---- final norm
  if ((rc = mark())) return rc;
  CK(launch_rmsnorm(h, 1, w->final_norm, h_out, dt, M, (int)d, sh->norm_eps, s), "final norm");
  if ((rc = mark())) return rc;
  return HDF_OK;
}

}  // namespace

extern "C" {

size_t hdf_draft_block_workspace_size(const hdf_draft_shape* shape) {
  if (check_draft_shape(shape) != HDF_OK) return 0;
  return draft_layout(shape).total;
}

int hdf_draft_block_workspace_layout(const hdf_draft_shape* shape, hdf_draft_workspace_layout* out) {
  g_err.clear();
  int rc = check_draft_shape(shape);
  if (rc) return rc;
  if (!out) return fail(HDF_ERR_INVALID_ARG, "out is NULL");
  const DraftLayout L = draft_layout(shape);
  out->c = L.c;
  out->k_ctx = L.kc;
  out->v_ctx = L.vc;
  out->h = L.h;
  out->x = L.x;
  out->q = L.q;
  out->k_blk = L.kb;
  out->v_blk = L.vb;
  out->o = L.o;
  out->act = L.act;
  out->total = L.total;
  return HDF_OK;
}

int hdf_draft_block(const hdf_drafter_weights* w, const hdf_draft_shape* sh, const void* ctx,
                    const int32_t* cu_ctx, const int32_t* anchor, void* h_out, void* ws, size_t ws_bytes,
                    const hdf_trace* trace, hdf_stream_t stream) {
  g_err.clear();
  int rc = check_draft_shape(sh);
  if (rc) return rc;
  if ((rc = check_drafter_weights(w, sh))) return rc;
  if ((long long)sh->batch * sh->block == 0) return HDF_OK;
  if (!cu_ctx || !anchor || !h_out || (sh->n_ctx > 0 && !ctx)) return fail(HDF_ERR_INVALID_ARG, "null input");
  if (w->rope_max_pos < (long long)sh->max_ctx + sh->block)
    return fail(HDF_ERR_SHAPE, "rope_max_pos %lld < max_ctx + block", (long long)w->rope_max_pos);
  if ((ctx && !aligned16(ctx)) || !aligned16(h_out)) return fail(HDF_ERR_ALIGNMENT, "tensor not 16-byte aligned");
  return draft_forward(w, sh, ctx, cu_ctx, nullptr, anchor, h_out, ws, ws_bytes, trace, (cudaStream_t)stream);
}

size_t hdf_draft_block_cached_workspace_size(const hdf_draft_shape* shape) {
  if (check_draft_shape(shape) != HDF_OK) return 0;
  hdf_draft_shape s = *shape;
  s.n_ctx = 0;
  return draft_layout(&s).total;
}

int hdf_draft_block_cached(const hdf_drafter_weights* w, const hdf_draft_shape* sh, const hdf_ctx_cache* cache,
                           const int32_t* anchor, void* h_out, void* ws, size_t ws_bytes, const hdf_trace* trace,
                           hdf_stream_t stream) {
  g_err.clear();
  int rc = check_draft_shape(sh);
  if (rc) return rc;
  if ((rc = check_drafter_weights(w, sh))) return rc;
  if ((rc = check_cache(cache, sh))) return rc;
  if (sh->max_ctx > cache->capacity)
    return fail(HDF_ERR_SHAPE, "max_ctx %d > cache capacity %d", sh->max_ctx, cache->capacity);
  if ((long long)sh->batch * sh->block == 0) return HDF_OK;
  if (!anchor || !h_out) return fail(HDF_ERR_INVALID_ARG, "null input");
  if (!aligned16(h_out)) return fail(HDF_ERR_ALIGNMENT, "h_out not 16-byte aligned");
  if (w->rope_max_pos < (long long)sh->max_ctx + sh->block)
    return fail(HDF_ERR_SHAPE, "rope_max_pos %lld < max_ctx + block", (long long)w->rope_max_pos);
  return draft_forward(w, sh, nullptr, nullptr, cache, anchor, h_out, ws, ws_bytes, trace, (cudaStream_t)stream);
}

size_t hdf_ctx_append_workspace_size(const hdf_draft_shape* shape) {
  if (check_draft_shape(shape) != HDF_OK) return 0;
  return std::max<size_t>(256, up256((size_t)shape->n_ctx * shape->d * esize(shape->dtype)));
}

int hdf_ctx_append(const hdf_drafter_weights* w, const hdf_draft_shape* sh, const void* ctx_new,
                   const int32_t* cu_new, const hdf_ctx_cache* cache, void* ws, size_t ws_bytes,
                   hdf_stream_t stream) {
  g_err.clear();
  int rc = check_draft_shape(sh);
  if (rc) return rc;
  if ((rc = check_drafter_weights(w, sh))) return rc;
  if ((rc = check_cache(cache, sh))) return rc;
  if (sh->batch == 0 || sh->n_ctx == 0) return HDF_OK;
  if (!ctx_new || !cu_new) return fail(HDF_ERR_INVALID_ARG, "ctx_new / cu_new NULL");
  if (!aligned16(ctx_new)) return fail(HDF_ERR_ALIGNMENT, "ctx_new not 16-byte aligned");
  if (w->rope_max_pos < cache->capacity)
    return fail(HDF_ERR_SHAPE, "rope_max_pos %lld < cache capacity %d", (long long)w->rope_max_pos, cache->capacity);
  const size_t need = hdf_ctx_append_workspace_size(sh);
  if (!ws || ws_bytes < need || (reinterpret_cast<uintptr_t>(ws) & 255))
    return fail(HDF_ERR_WORKSPACE, "workspace %zu bytes (need %zu, 256-byte aligned)", ws_bytes, need);
  cudaStream_t s = (cudaStream_t)stream;
  const AppendIn ap{ctx_new, cu_new, sh->n_ctx, ws};
  if ((rc = append_rows(w, sh, ap, cache, s))) return rc;
  CK(launch_cache_advance(cache->len, cu_new, sh->batch, cache->capacity, device_status_ptr(), s), "cache advance");
  return HDF_OK;
}

size_t hdf_draft_round_workspace_size(const hdf_draft_shape* shape) {
  if (check_draft_shape(shape) != HDF_OK) return 0;
  return hdf_ctx_append_workspace_size(shape) + hdf_draft_block_cached_workspace_size(shape);
}

int hdf_draft_round(const hdf_drafter_weights* w, const hdf_draft_shape* sh, const void* ctx_new,
                    const int32_t* cu_new, const hdf_ctx_cache* cache, const int32_t* anchor, void* h_out, void* ws,
                    size_t ws_bytes, hdf_stream_t stream) {
  g_err.clear();
  int rc = check_draft_shape(sh);
  if (rc) return rc;
  if ((rc = check_drafter_weights(w, sh))) return rc;
  if ((rc = check_cache(cache, sh))) return rc;
  const long long n_new = sh->batch > 0 ? sh->n_ctx : 0;
  const bool has_block = (long long)sh->batch * sh->block > 0;
  if (n_new == 0 && !has_block) return HDF_OK;
  if (n_new > 0) {
    if (!ctx_new || !cu_new) return fail(HDF_ERR_INVALID_ARG, "ctx_new / cu_new NULL");
    if (!aligned16(ctx_new)) return fail(HDF_ERR_ALIGNMENT, "ctx_new not 16-byte aligned");
    if (w->rope_max_pos < cache->capacity)
      return fail(HDF_ERR_SHAPE, "rope_max_pos %lld < cache capacity %d", (long long)w->rope_max_pos,
                  cache->capacity);
  }
  if (has_block) {
    if (sh->max_ctx > cache->capacity)
      return fail(HDF_ERR_SHAPE, "max_ctx %d > cache capacity %d", sh->max_ctx, cache->capacity);
    if (!anchor || !h_out) return fail(HDF_ERR_INVALID_ARG, "null input");
    if (!aligned16(h_out)) return fail(HDF_ERR_ALIGNMENT, "h_out not 16-byte aligned");
    if (w->rope_max_pos < (long long)sh->max_ctx + sh->block)
      return fail(HDF_ERR_SHAPE, "rope_max_pos %lld < max_ctx + block", (long long)w->rope_max_pos);
  }
  const size_t need_a = hdf_ctx_append_workspace_size(sh);
  const size_t need = hdf_draft_round_workspace_size(sh);
  if (!ws || ws_bytes < need || (reinterpret_cast<uintptr_t>(ws) & 255))
    return fail(HDF_ERR_WORKSPACE, "workspace %zu bytes (need %zu, 256-byte aligned)", ws_bytes, need);
  cudaStream_t s = (cudaStream_t)stream;
  const AppendIn ap{ctx_new, cu_new, n_new, ws};
  if (!has_block) {  // nothing to draft: the append alone
    if ((rc = append_rows(w, sh, ap, cache, s))) return rc;
    CK(launch_cache_advance(cache->len, cu_new, sh->batch, cache->capacity, device_status_ptr(), s), "cache advance");
    return HDF_OK;
  }
  return draft_forward(w, sh, nullptr, nullptr, cache, anchor, h_out, static_cast<char*>(ws) + need_a,
                       ws_bytes - need_a, nullptr, s, &ap);
}

// -------------------------------------------------------------- LM head
namespace {
struct LmLayout {
  SplitPlan p;
  bool token_major;
  int tiles;    // vocabulary tiles the partials come from
  int tiles_m;
  size_t pmax, parg, psum, total;
};
// Token-major LM head (tokens on the GEMM rows, 224 or 256 vocabulary columns
// per tile) from this many tokens: each CTA then streams about 1.5 bytes per
// weight byte instead of 2 (the swapped tile re-reads a token tile as large
// as its weight tile)
constexpr int64_t kLmTokenMajorFrom = 64;

// Vocabulary columns per token-major tile: of 256 and 224, the one with the
// least waves x width over two resident CTAs per SM.  At V = 129,280 and
// 128 tokens: 505 tiles of 256 take 1.66 waves (2 x 256), 578 tiles of 224
// take 1.90 (2 x 224).
int lm_token_major_bn(int64_t M, int64_t V) {
  const long long slots = 2LL * num_sms(), tm = (M + 127) / 128;
  int best = 256;
  long long best_cost = LLONG_MAX;
  for (int bn : {256, 224}) {
    const long long tiles = tm * ((V + bn - 1) / bn);
    const long long cost = (tiles + slots - 1) / slots * bn;
    if (cost < best_cost) {
      best_cost = cost;
      best = bn;
    }
  }
  return best;
}

LmLayout lm_layout(int64_t M, int64_t V, int dtype, int d) {
  LmLayout L;
  L.token_major = M >= kLmTokenMajorFrom;
  const int tbn = L.token_major ? lm_token_major_bn(M, V) : 0;
  L.p = L.token_major ? SplitPlan{tbn, 1, (int)(((M + 127) / 128) * ((V + tbn - 1) / tbn))} : plan_swap(dtype, V, M, d);
  L.tiles_m = (int)((V + 127) / 128);  // partial rows reserved: enough for either orientation
  L.tiles = L.token_major ? (int)((V + tbn - 1) / tbn) : L.tiles_m;
  size_t off = 0;
  auto take = [&](size_t b) {
    const size_t o = off;
    off += up256(b);
    return o;
  };
  L.pmax = take((size_t)L.tiles_m * M * 4);
  L.parg = take((size_t)L.tiles_m * M * 4);
  L.psum = take((size_t)L.tiles_m * M * 4);
  L.total = off;
  return L;
}

// LM-head GEMM with the argmax / sum-exp epilogue, then the cross-tile reduce.
int lm_head_launch(const LmLayout& L, const void* h, int dtype, int64_t M, int d, const void* W_lm, int64_t V,
                   float inv_temp, int32_t* tok, float* zmax, float* logsoftmax, char* W, cudaStream_t s) {
  GemmArgs g;
  int rc;
  if (L.token_major) {
    init_gemm(g, dtype, M, V, d, L.p);
    g.group_n = 8;  // the token tiles of one weight tile run together
    if ((rc = make_map(&g.A.map[0], h, dtype, M, d, d, 64))) return rc;
    if ((rc = make_map(&g.B.map[0], W_lm, dtype, V, d, d, L.p.bn))) return rc;
    g.pre_operand = 2;  // the LM head weight
    g.epi.kind = kEpiLmHead;
  } else {
    init_gemm(g, dtype, V, M, d, L.p);
    if ((rc = make_map(&g.A.map[0], W_lm, dtype, V, d, d, 64))) return rc;
    if ((rc = make_map(&g.B.map[0], h, dtype, M, d, d, L.p.bn))) return rc;
    g.pre_operand = 1;  // the LM head weight
    g.epi.kind = kEpiLmHeadT;
  }
  g.epi.inv_temp = inv_temp;
  g.epi.logsoftmax = logsoftmax;
  g.epi.part_max = reinterpret_cast<float*>(W + L.pmax);
  g.epi.part_arg = reinterpret_cast<int*>(W + L.parg);
  g.epi.part_sum = reinterpret_cast<float*>(W + L.psum);
  CK(launch_gemm(g, s), "lm head gemm");
  CK(launch_lm_reduce(g.epi.part_max, g.epi.part_arg, g.epi.part_sum, L.tiles, M, V, inv_temp, tok, zmax,
                      logsoftmax, s),
     "lm reduce");
  return HDF_OK;
}
}  // namespace

size_t hdf_lm_head_workspace_size(int64_t M, int d, int64_t V, int dtype) {
  if (M <= 0 || V <= 0 || d <= 0) return 0;
  return lm_layout(M, V, dtype, d).total;
}

int hdf_lm_head_argmax(const void* h, int dtype, int64_t M, int d, const void* W_lm, int64_t V, float inv_temp,
                       int32_t* tok, float* zmax, float* logsoftmax, void* ws, size_t ws_bytes,
                       hdf_stream_t stream) {
  g_err.clear();
  if (dtype != HDF_BF16 && dtype != HDF_F32) return fail(HDF_ERR_DTYPE, "dtype %d", dtype);
  if (M < 0 || V <= 0 || d <= 0 || d > 65536 || V > 0x7fffffffLL || M > 0x7fffffffLL)
    return fail(HDF_ERR_SHAPE, "M/V/d");
  if ((d * esize(dtype)) % 16) return fail(HDF_ERR_SHAPE, "d row stride must be a multiple of 16 bytes");
  if (!(inv_temp > 0) || !std::isfinite(inv_temp)) return fail(HDF_ERR_INVALID_ARG, "inv_temp must be > 0");
  if (M == 0) return HDF_OK;
  if (!h || !W_lm || !tok) return fail(HDF_ERR_INVALID_ARG, "null pointer");
  if (!aligned16(h) || !aligned16(W_lm)) return fail(HDF_ERR_ALIGNMENT, "h / W_lm alignment");
  const LmLayout L = lm_layout(M, V, dtype, d);
  if (!ws || ws_bytes < L.total || (reinterpret_cast<uintptr_t>(ws) & 255))
    return fail(HDF_ERR_WORKSPACE, "workspace %zu bytes (need %zu, 256-byte aligned)", ws_bytes, L.total);
  return lm_head_launch(L, h, dtype, M, d, W_lm, V, inv_temp, tok, zmax, logsoftmax, static_cast<char*>(ws),
                        (cudaStream_t)stream);
}

// ------------------------------------------------ T = 1 verification
int hdf_accept_sample(const float* p_target, const float* q_draft, const int32_t* draft, int64_t draft_stride,
                      const uint32_t* u, const uint32_t* r, int batch, int n_draft, int64_t V, int32_t* accept,
                      int32_t* next_tok, hdf_stream_t stream) {
  g_err.clear();
  if (batch < 0 || n_draft < 0 || V < 1 || V > ((int64_t)1 << 22))
    return fail(HDF_ERR_SHAPE, "batch / n_draft / V (1..2^22)");
  if (batch == 0) return HDF_OK;
  if (n_draft > 0 && draft_stride < n_draft) return fail(HDF_ERR_SHAPE, "draft_stride < n_draft");
  if (!p_target || !r || !accept || !next_tok || (n_draft > 0 && (!q_draft || !draft || !u)))
    return fail(HDF_ERR_INVALID_ARG, "null pointer");
  CK(launch_accept_sample(p_target, q_draft, draft, draft_stride, u, r, batch, n_draft, V, accept, next_tok,
                          (cudaStream_t)stream),
     "accept sample");
  return HDF_OK;
}

// ----------------------------------------------------- KL distillation
size_t hdf_kl_distill_workspace_size(int64_t rows, int64_t V) {
  if (rows <= 0 || V <= 0) return 0;
  return up256((size_t)rows * kl_chunks(V) * 4);
}

int hdf_kl_distill(const float* ls_teacher, const float* ls_student, int64_t rows, int64_t V, float t_kd,
                   float* kl_rows, float* kl_mean, void* ws, size_t ws_bytes, hdf_stream_t stream) {
  g_err.clear();
  if (rows < 0 || V <= 0 || rows > 65535 || V > ((int64_t)1 << 40)) return fail(HDF_ERR_SHAPE, "rows / V");
  if (!(t_kd > 0) || !std::isfinite(t_kd)) return fail(HDF_ERR_INVALID_ARG, "t_kd must be > 0");
  if (rows == 0) return HDF_OK;
  if (!ls_teacher || !ls_student) return fail(HDF_ERR_INVALID_ARG, "ls_teacher and ls_student are required");
  if (!aligned16(ls_teacher) || !aligned16(ls_student))
    return fail(HDF_ERR_ALIGNMENT, "ls_teacher and ls_student must be 16-byte aligned");
  const size_t need = hdf_kl_distill_workspace_size(rows, V);
  if (!ws || ws_bytes < need || (reinterpret_cast<uintptr_t>(ws) & 255))
    return fail(HDF_ERR_WORKSPACE, "workspace %zu bytes (need %zu, 256-byte aligned)", ws_bytes, need);
  CK(launch_kl_distill(ls_teacher, ls_student, rows, V, t_kd, kl_rows, kl_mean, static_cast<float*>(ws),
                       (cudaStream_t)stream),
     "kl distill");
  return HDF_OK;
}

// ------------------------------------------------ training objective, Eq. 3
size_t hdf_draft_loss_workspace_size(int batch, int P, int64_t V) {
  if (batch <= 0 || P <= 0 || V <= 0) return 0;
  return up256((size_t)loss_partial_floats(batch, P, V) * 4);
}

int hdf_draft_loss(const float* ls_teacher, const float* ls_student, const int32_t* labels, int batch, int block,
                   int P, int64_t V, float t_kd, float alpha, float* ce_rows, float* kl_rows, float* loss, void* ws,
                   size_t ws_bytes, hdf_stream_t stream) {
  g_err.clear();
  if (batch < 0 || block < 2 || block > 64 || P < 0 || P > block - 1 || V <= 0 || V > ((int64_t)1 << 31))
    return fail(HDF_ERR_SHAPE, "need batch >= 0, 2 <= block <= 64, 0 <= P <= block - 1, 0 < V <= 2^31 (batch %d, "
                "block %d, P %d, V %lld)", batch, block, P, (long long)V);
  if ((int64_t)batch * block > 65535) return fail(HDF_ERR_SHAPE, "batch * block above 65535");
  if (!(t_kd > 0) || !std::isfinite(t_kd)) return fail(HDF_ERR_INVALID_ARG, "t_kd must be finite and > 0");
  if (!std::isfinite(alpha)) return fail(HDF_ERR_INVALID_ARG, "alpha must be finite");
  if (batch == 0) return HDF_OK;
  if (!ls_student || !labels || !loss || (P > 0 && !ls_teacher))
    return fail(HDF_ERR_INVALID_ARG, "ls_student, labels, loss (and ls_teacher when P > 0) are required");
  if (!aligned16(ls_student) || (P > 0 && !aligned16(ls_teacher)))
    return fail(HDF_ERR_ALIGNMENT, "ls_teacher and ls_student must be 16-byte aligned");
  const size_t need = hdf_draft_loss_workspace_size(batch, P, V);
  if (need && (!ws || ws_bytes < need || (reinterpret_cast<uintptr_t>(ws) & 255)))
    return fail(HDF_ERR_WORKSPACE, "workspace %zu bytes (need %zu, 256-byte aligned)", ws_bytes, need);
  CK(launch_draft_loss(ls_teacher, ls_student, labels, batch, block, P, V, t_kd, alpha, ce_rows, kl_rows, loss,
                       static_cast<float*>(ws), device_status_ptr(), (cudaStream_t)stream),
     "draft loss");
  return HDF_OK;
}

// ------------------------------------------ LM head on library-owned scratch
// For callers that cannot allocate device memory themselves: the LM head's
// scratch (per-tile argmax / sum-exp partials) lives in this file-scope device array instead of a caller
// workspace.  Every GPU that loads the library holds the array until the
// process exits; all calls share it.
}  // extern "C"
namespace {
__device__ __align__(256) unsigned char g_lm_static_scratch[HDF_LM_HEAD_STATIC_SCRATCH_BYTES];
static_assert(HDF_LM_HEAD_STATIC_SCRATCH_BYTES % 256 == 0, "scratch size must keep 256-byte alignment");

// Device address of the scratch array on the current device.  In host code
// the array's name is only a host-side stand-in, so the address has to come
// from cudaGetSymbolAddress, once per device, with that device current.
int lm_static_scratch(void** out) {
  static std::mutex mu;
  static void* ptr[64] = {nullptr};
  int dev = 0;
  CK(cudaGetDevice(&dev), "cudaGetDevice");
  if (dev < 0 || dev >= 64) return fail(HDF_ERR_UNSUPPORTED, "device ordinal %d", dev);
  std::lock_guard<std::mutex> lock(mu);
  if (!ptr[dev]) {
    void* p = nullptr;
    CK(cudaGetSymbolAddress(&p, g_lm_static_scratch), "cudaGetSymbolAddress(LM-head scratch)");
    ptr[dev] = p;
  }
  *out = ptr[dev];
  return HDF_OK;
}
}  // namespace
extern "C" {

int hdf_lm_head_argmax_static(const void* h, int dtype, int64_t M, int d, const void* W_lm, int64_t V,
                              float inv_temp, int32_t* tok, float* zmax, float* logsoftmax, hdf_stream_t stream) {
  g_err.clear();
  const bool sizes_ok = (dtype == HDF_BF16 || dtype == HDF_F32) && M > 0 && V > 0 && d > 0 && d <= 65536 &&
                        V <= 0x7fffffffLL && M <= 0x7fffffffLL;
  if (!sizes_ok)  // let the workspace entry point report the exact argument error (or M == 0: nothing to do)
    return hdf_lm_head_argmax(h, dtype, M, d, W_lm, V, inv_temp, tok, zmax, logsoftmax, nullptr, 0, stream);
  const size_t need = lm_layout(M, V, dtype, d).total;
  if (need > (size_t)HDF_LM_HEAD_STATIC_SCRATCH_BYTES)
    return fail(HDF_ERR_WORKSPACE,
                "M=%lld d=%d V=%lld needs %zu bytes of scratch, the library's static buffer holds %zu; "
                "use hdf_lm_head_argmax with a caller workspace",
                (long long)M, d, (long long)V, need, (size_t)HDF_LM_HEAD_STATIC_SCRATCH_BYTES);
  void* ws = nullptr;
  int rc = lm_static_scratch(&ws);
  if (rc) return rc;
  // nothing in the shared array needs clearing between calls: the GEMM
  // epilogue writes every [tile, row] partial (max, argmax, sum-exp) of this
  // call before lm_reduce_kernel, the next kernel in the stream, reads it
  return hdf_lm_head_argmax(h, dtype, M, d, W_lm, V, inv_temp, tok, zmax, logsoftmax, ws,
                            (size_t)HDF_LM_HEAD_STATIC_SCRATCH_BYTES, stream);
}

// -------------------------------------------------------------- verify
int hdf_accept_len(const int32_t* draft, int64_t draft_stride, const int32_t* target, int64_t target_stride,
                   int batch, int n_draft, int32_t* accept, hdf_stream_t stream) {
  g_err.clear();
  if (batch < 0 || n_draft < 0) return fail(HDF_ERR_SHAPE, "batch/n_draft");
  if (n_draft > 47) return fail(HDF_ERR_UNSUPPORTED, "n_draft %d > 47", n_draft);
  if (batch == 0) return HDF_OK;
  if (!draft || !target || !accept) return fail(HDF_ERR_INVALID_ARG, "null pointer");
  if (draft_stride < n_draft || target_stride < n_draft) return fail(HDF_ERR_SHAPE, "stride < n_draft");
  CK(launch_accept(draft, draft_stride, target, target_stride, batch, n_draft, accept, (cudaStream_t)stream),
     "accept launch");
  return HDF_OK;
}

}  // extern "C"
