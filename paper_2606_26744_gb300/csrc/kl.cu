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

}  // namespace

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
