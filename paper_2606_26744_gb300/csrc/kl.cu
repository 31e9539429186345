// KL distillation target, Eq. 2 of the HyperDFlash paper (Sec. 2.3):
//   KL(p || q) = sum_v p(v) * (log p(v) - log q(v)),  L_KL = T^2 / rows * sum_rows KL
// over log-softmax rows at temperature T.  Memory-bound: both inputs are
// read once with 16-byte loads.  Stage 1 spreads every row over chunks of
// KL_CHUNK entries (one CTA per chunk and row) and writes one partial sum per
// CTA; stage 2 (one CTA) adds the partials of each row in chunk order and the
// rows in row order, so the result does not depend on scheduling.
#include "common.cuh"
#include "kernels.h"

namespace hdf {
namespace {

constexpr int KL_THREADS = 256;

__device__ __forceinline__ float kl_term(float lp, float lq) {
  // a teacher entry of -inf has p = 0 and contributes nothing (0 * inf is not taken)
  return lp == -INFINITY ? 0.f : expf(lp) * (lp - lq);
}

// Fixed-order sum of one value per thread of the CTA.
__device__ __forceinline__ float block_sum_fixed(float v, float* sh) {
  v = warp_sum(v);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (lane == 0) sh[warp] = v;
  __syncthreads();
  float s = 0.f;
  if (threadIdx.x == 0)
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) s += sh[w];
  return s;  // valid in thread 0
}

__global__ void __launch_bounds__(KL_THREADS) kl_partial_kernel(const float* __restrict__ lt,
                                                                const float* __restrict__ ls, long long V,
                                                                int nchunks, float* __restrict__ partial) {
  __shared__ float sh[KL_THREADS / 32];
  pdl_launch_dependents();
  pdl_wait();
  const int chunk = blockIdx.x;
  const long long row = blockIdx.y;
  const long long v0 = (long long)chunk * KL_CHUNK, v1 = min(V, v0 + KL_CHUNK);
  const float* a = lt + row * V;
  const float* b = ls + row * V;
  float acc = 0.f;
  if ((V & 3) == 0) {  // rows are 16-byte aligned: float4 loads, all of a thread's loads issued first
    constexpr int PER = KL_CHUNK / (4 * KL_THREADS);
    float4 x[PER], y[PER];
#pragma unroll
    for (int i = 0; i < PER; ++i) {
      const long long v = v0 + 4 * ((long long)i * KL_THREADS + threadIdx.x);
      const bool in = v < v1;  // chunks start on multiples of 4, so a vector is wholly in or out
      x[i] = in ? __ldcs(reinterpret_cast<const float4*>(a + v)) : make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
      y[i] = in ? __ldcs(reinterpret_cast<const float4*>(b + v)) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int i = 0; i < PER; ++i)
      acc += (kl_term(x[i].x, y[i].x) + kl_term(x[i].y, y[i].y)) + (kl_term(x[i].z, y[i].z) + kl_term(x[i].w, y[i].w));
  } else {
    for (long long v = v0 + threadIdx.x; v < v1; v += KL_THREADS) acc += kl_term(a[v], b[v]);
  }
  const float s = block_sum_fixed(acc, sh);
  if (threadIdx.x == 0) partial[row * nchunks + chunk] = s;
}

__global__ void __launch_bounds__(KL_THREADS) kl_final_kernel(const float* __restrict__ partial, long long rows,
                                                              int nchunks, float scale, float* kl_rows,
                                                              float* kl_mean) {
  __shared__ float sh[KL_THREADS / 32];
  pdl_launch_dependents();
  pdl_wait();
  float mine = 0.f;
  for (long long r = threadIdx.x; r < rows; r += KL_THREADS) {
    float s = 0.f;
    for (int c = 0; c < nchunks; ++c) s += partial[r * nchunks + c];
    if (kl_rows) kl_rows[r] = s;
    mine += s;
  }
  const float total = block_sum_fixed(mine, sh);
  if (threadIdx.x == 0 && kl_mean) *kl_mean = scale * total;
}

// ---------------------------------------------------------------------------
// Training objective of Eq. 3, L = L_CE + alpha * L_KL, over a batch of
// blocks.  Both inputs are log-softmax rows at temperature 1; the KL part
// needs the softmaxes at T_KD, softmax(ls / T_KD), whose normaliser is not
// known in advance.  Stage 1 takes, per (row, chunk), in one pass over the
// two rows (x = teacher * it, y = student * it, it = 1 / T_KD):
//   mx = max x,  sx = sum e^(x - mx),  w = sum e^(x - mx) * (x - y),
//   my = max y,  sy = sum e^(y - my).
// Merged over the chunks in chunk order, KL(p || q) = w / sx - (mx + log sx)
// + (my + log sy): the sum of p * (log p - log q) with log p = x - lse(x),
// log q = y - lse(y).  For identical rows w is exactly 0 and the two
// normalisers are the same computation, so the KL is exactly 0.
struct Lse5 {
  float mx, sx, w, my, sy;
};

__device__ __forceinline__ float rescale(float m_old, float m_new) {
  // e^(m_old - m_new); a part that saw only -inf has nothing to rescale
  return m_old == -INFINITY ? 0.f : expf(m_old - m_new);
}

__device__ __forceinline__ Lse5 lse5_merge(const Lse5& a, const Lse5& b) {
  Lse5 r;
  r.mx = fmaxf(a.mx, b.mx);
  const float fa = rescale(a.mx, r.mx), fb = rescale(b.mx, r.mx);
  r.sx = a.sx * fa + b.sx * fb;
  r.w = a.w * fa + b.w * fb;
  r.my = fmaxf(a.my, b.my);
  r.sy = a.sy * rescale(a.my, r.my) + b.sy * rescale(b.my, r.my);
  return r;
}

constexpr int LOSS_PER = KL_CHUNK / (4 * KL_THREADS);  // float4 loads per thread and row

__global__ void __launch_bounds__(KL_THREADS) loss_kl_partial_kernel(const float* __restrict__ lt,
                                                                     const float* __restrict__ ls, long long V,
                                                                     int block, int P, float it, int nchunks,
                                                                     Lse5* __restrict__ partial) {
  __shared__ Lse5 sh[KL_THREADS / 32];
  pdl_launch_dependents();
  pdl_wait();
  const int chunk = blockIdx.x;
  const long long r = blockIdx.y;                 // teacher row: block r / P, position k = r % P + 1
  const long long srow = (r / P) * block + r % P + 1;
  const long long v0 = (long long)chunk * KL_CHUNK, v1 = min(V, v0 + KL_CHUNK);
  const float* a = lt + r * V;
  const float* b = ls + srow * V;
  // every value of this thread's slice of the chunk, loaded before any arithmetic
  float x[4 * LOSS_PER], y[4 * LOSS_PER];
  if ((V & 3) == 0) {  // 16-byte rows: float4 loads; chunks start on multiples of 4
#pragma unroll
    for (int i = 0; i < LOSS_PER; ++i) {
      const long long v = v0 + 4 * ((long long)i * KL_THREADS + threadIdx.x);
      const bool in = v < v1;
      const float4 p = in ? __ldcs(reinterpret_cast<const float4*>(a + v))
                          : make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
      const float4 q = in ? __ldcs(reinterpret_cast<const float4*>(b + v))
                          : make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
      x[4 * i] = p.x, x[4 * i + 1] = p.y, x[4 * i + 2] = p.z, x[4 * i + 3] = p.w;
      y[4 * i] = q.x, y[4 * i + 1] = q.y, y[4 * i + 2] = q.z, y[4 * i + 3] = q.w;
    }
  } else {
#pragma unroll
    for (int i = 0; i < 4 * LOSS_PER; ++i) {
      const long long v = v0 + (long long)i * KL_THREADS + threadIdx.x;
      x[i] = v < v1 ? a[v] : -INFINITY;
      y[i] = v < v1 ? b[v] : -INFINITY;
    }
  }
  Lse5 acc{-INFINITY, 0.f, 0.f, -INFINITY, 0.f};
#pragma unroll
  for (int i = 0; i < 4 * LOSS_PER; ++i) {
    x[i] *= it;
    y[i] *= it;
    acc.mx = fmaxf(acc.mx, x[i]);
    acc.my = fmaxf(acc.my, y[i]);
  }
#pragma unroll
  for (int i = 0; i < 4 * LOSS_PER; ++i) {
    if (x[i] != -INFINITY) {  // p = 0 contributes nothing (0 * inf is not taken)
      const float e = expf(x[i] - acc.mx);
      acc.sx += e;
      acc.w += e * (x[i] - y[i]);
    }
    if (y[i] != -INFINITY) acc.sy += expf(y[i] - acc.my);
  }
  // fixed-order combine: butterfly within each warp, then the warps in order
  for (int off = 16; off > 0; off >>= 1) {
    Lse5 o{__shfl_xor_sync(0xffffffffu, acc.mx, off), __shfl_xor_sync(0xffffffffu, acc.sx, off),
           __shfl_xor_sync(0xffffffffu, acc.w, off), __shfl_xor_sync(0xffffffffu, acc.my, off),
           __shfl_xor_sync(0xffffffffu, acc.sy, off)};
    acc = lse5_merge(acc, o);
  }
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (lane == 0) sh[warp] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    Lse5 t = sh[0];
    for (int w = 1; w < KL_THREADS / 32; ++w) t = lse5_merge(t, sh[w]);
    partial[r * nchunks + chunk] = t;
  }
}

__global__ void __launch_bounds__(KL_THREADS) loss_final_kernel(const Lse5* __restrict__ partial,
                                                                const float* __restrict__ ls,
                                                                const int* __restrict__ labels, int batch,
                                                                int block, int P, long long V, int nchunks,
                                                                float kl_scale, float alpha, float* ce_rows,
                                                                float* kl_rows, float* loss, int* status) {
  __shared__ float sh[KL_THREADS / 32];
  __shared__ float cnt_sh[KL_THREADS / 32];
  pdl_launch_dependents();
  pdl_wait();
  // KL rows: chunks merged in chunk order, rows summed in row order per thread
  float kl_mine = 0.f;
  const long long n_kl = (long long)batch * P;
  for (long long r = threadIdx.x; r < n_kl; r += KL_THREADS) {
    Lse5 t = partial[r * nchunks];
    for (int c = 1; c < nchunks; ++c) t = lse5_merge(t, partial[r * nchunks + c]);
    const float kl = t.w / t.sx - (t.mx + logf(t.sx)) + (t.my + logf(t.sy));
    if (kl_rows) kl_rows[r] = kl;
    kl_mine += kl;
  }
  // CE rows: -log q_k(label) read from the student's log-softmax row
  float ce_mine = 0.f, n_mine = 0.f;
  const long long n_ce = (long long)batch * (block - 1);
  for (long long q = threadIdx.x; q < n_ce; q += KL_THREADS) {
    const long long i = q / (block - 1), k = q % (block - 1) + 1;
    const int lab = labels[q];
    float ce = __int_as_float(0x7fc00000);  // NaN: no supervision on this position
    if (lab >= 0 && lab < V) {
      ce = -ls[(i * block + k) * V + lab];
      ce_mine += ce;
      n_mine += 1.f;
    } else if (lab >= V) {
      record_device_error(status);  // a label outside the vocabulary: the position is left out
    }
    if (ce_rows) ce_rows[q] = ce;
  }
  const float kl_sum = block_sum_fixed(kl_mine, sh);
  __syncthreads();
  const float ce_sum = block_sum_fixed(ce_mine, sh);
  const float n_sup = block_sum_fixed(n_mine, cnt_sh);
  if (threadIdx.x == 0 && loss) {
    const float l_ce = n_sup > 0.f ? ce_sum / n_sup : 0.f;
    const float l_kl = kl_scale * kl_sum;
    loss[0] = l_ce + alpha * l_kl;
    loss[1] = l_ce;
    loss[2] = l_kl;
  }
}

}  // namespace

int loss_partial_floats(int batch, int P, long long V) { return batch * P * kl_chunks(V) * 5; }

cudaError_t launch_draft_loss(const float* lt, const float* ls, const int* labels, int batch, int block, int P,
                              long long V, float t_kd, float alpha, float* ce_rows, float* kl_rows, float* loss,
                              float* partial, int* status, cudaStream_t s) {
  if (batch == 0) return cudaSuccess;
  const int nc = kl_chunks(V);
  Lse5* part = reinterpret_cast<Lse5*>(partial);
  cudaError_t e = cudaSuccess;
  if (P > 0)
    e = launch_kernel(loss_kl_partial_kernel, dim3((unsigned)nc, (unsigned)(batch * P)), dim3(KL_THREADS), 0, s, 1u,
                      lt, ls, V, block, P, (float)(1.0 / (double)t_kd), nc, part);
  if (e != cudaSuccess) return e;
  const float kl_scale = P > 0 ? (float)((double)t_kd * t_kd / P / batch) : 0.f;
  return launch_kernel(loss_final_kernel, dim3(1), dim3(KL_THREADS), 0, s, 1u, (const Lse5*)part, ls, labels, batch,
                       block, P, V, nc, kl_scale, alpha, ce_rows, kl_rows, loss, status);
}

int kl_chunks(long long V) { return (int)((V + KL_CHUNK - 1) / KL_CHUNK); }

cudaError_t launch_kl_distill(const float* lt, const float* ls, long long rows, long long V, float t_kd,
                              float* kl_rows, float* kl_mean, float* partial, cudaStream_t s) {
  if (rows == 0) return cudaSuccess;
  const int nc = kl_chunks(V);
  cudaError_t e = launch_kernel(kl_partial_kernel, dim3((unsigned)nc, (unsigned)rows), dim3(KL_THREADS), 0, s, 1u,
                                lt, ls, V, nc, partial);
  if (e != cudaSuccess) return e;
  return launch_kernel(kl_final_kernel, dim3(1), dim3(KL_THREADS), 0, s, 1u, partial, rows, nc,
                       t_kd * t_kd / (float)rows, kl_rows, kl_mean);
}

}  // namespace hdf
