// Small kernels of the draft step: RoPE tables, RMSNorm, block embedding,
// block verification (accepted-prefix length) and the cross-tile LM-head
// reduction (argmax / log-sum-exp / log-softmax).
#include <climits>
#include <cmath>

#include "common.cuh"
#include "kernels.h"

namespace hdf {
namespace {

// cos/sin of p * theta^(-2i/hd) in double precision, stored fp32.
__global__ void rope_table_kernel(double theta, int hd, long long max_pos, float* c, float* s) {
  const int half = hd / 2;
  const long long n = max_pos * half;
  for (long long k = blockIdx.x * (long long)blockDim.x + threadIdx.x; k < n;
       k += (long long)gridDim.x * blockDim.x) {
    const long long p = k / half;
    const int i = (int)(k - p * half);
    const double inv_freq = pow(theta, -2.0 * (double)i / (double)hd);
    double sn, cs;
    sincos((double)p * inv_freq, &sn, &cs);
    c[k] = (float)cs;
    s[k] = (float)sn;
  }
}

__device__ __forceinline__ float block_sum(float v, float* sh) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  v = warp_sum(v);
  if (lane == 0) sh[warp] = v;
  __syncthreads();
  float t = 0.f;
  const int nw = blockDim.x >> 5;
  for (int w = 0; w < nw; ++w) t += sh[w];
  __syncthreads();
  return t;
}

// One CTA per row: y = x / sqrt(mean(x^2) + eps) * w.  x is XT, y is T.
template <typename XT, typename T>
__global__ void rmsnorm_kernel(const XT* __restrict__ x, const T* __restrict__ w, T* __restrict__ y,
                               int d, float eps) {
  __shared__ float sh[32];
  const long long r = blockIdx.x;
  const XT* xr = x + r * d;
  float ss = 0.f;
  for (int i = threadIdx.x; i < d; i += blockDim.x) {
    const float v = to_f32(xr[i]);
    ss = fmaf(v, v, ss);
  }
  const float inv = rsqrtf(block_sum(ss, sh) / (float)d + eps);
  T* yr = y + r * d;
  for (int i = threadIdx.x; i < d; i += blockDim.x) yr[i] = from_f32<T>(to_f32(xr[i]) * inv * to_f32(w[i]));
}

// Vectorised bf16 -> bf16 RMSNorm (context rows): 16-byte loads and stores.
__global__ void rmsnorm_bf16_vec_kernel(const __nv_bfloat16* __restrict__ x,
                                        const __nv_bfloat16* __restrict__ w,
                                        __nv_bfloat16* __restrict__ y, int d, float eps) {
  __shared__ float sh[32];
  const long long r = blockIdx.x;
  const int nv = d / 8;
  const uint4* xr = reinterpret_cast<const uint4*>(x + r * d);
  float ss = 0.f;
  for (int i = threadIdx.x; i < nv; i += blockDim.x) {
    float f[8];
    V16<__nv_bfloat16>::unpack(ld_stream16(xr + i), f);
#pragma unroll
    for (int e = 0; e < 8; ++e) ss = fmaf(f[e], f[e], ss);
  }
  const float inv = rsqrtf(block_sum(ss, sh) / (float)d + eps);
  uint4* yr = reinterpret_cast<uint4*>(y + r * d);
  const uint4* wr = reinterpret_cast<const uint4*>(w);
  for (int i = threadIdx.x; i < nv; i += blockDim.x) {
    float f[8], g[8];
    V16<__nv_bfloat16>::unpack(ld_nc16(xr + i), f);
    V16<__nv_bfloat16>::unpack(ld_nc16(wr + i), g);
#pragma unroll
    for (int e = 0; e < 8; ++e) f[e] = f[e] * inv * g[e];
    yr[i] = V16<__nv_bfloat16>::pack(f);
  }
}

// Block input [anchor; mask x (B-1)] into the fp32 residual, then RMSNorm.
template <typename T>
__global__ void embed_norm_kernel(const T* __restrict__ embed, const T* __restrict__ mask_vec,
                                  const int* __restrict__ anchor, const T* __restrict__ w,
                                  float* __restrict__ h, T* __restrict__ x, int block, int d, int vocab,
                                  float eps) {
  __shared__ float sh[32];
  const int r = blockIdx.x;
  const int i = r / block, k = r - i * block;
  const int tokid = min(max(__ldg(anchor + i), 0), vocab - 1);  // ids outside [0, V) are clamped
  const T* src = k == 0 ? embed + (long long)tokid * d : mask_vec;
  float ss = 0.f;
  for (int e = threadIdx.x; e < d; e += blockDim.x) {
    const float v = to_f32(src[e]);
    h[(long long)r * d + e] = v;
    ss = fmaf(v, v, ss);
  }
  const float inv = rsqrtf(block_sum(ss, sh) / (float)d + eps);
  for (int e = threadIdx.x; e < d; e += blockDim.x)
    x[(long long)r * d + e] = from_f32<T>(to_f32(src[e]) * inv * to_f32(w[e]));
}

__global__ void accept_kernel(const int* __restrict__ draft, long long ds, const int* __restrict__ target,
                              long long ts, int batch, int nd, int* __restrict__ accept) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= batch) return;
  int n = 0;
  while (n < nd && draft[(long long)i * ds + n] == target[(long long)i * ts + n]) ++n;
  accept[i] = n;
}

struct MaxArgSum {
  float m;
  int a;
  float s;
};
__device__ __forceinline__ MaxArgSum combine(MaxArgSum x, MaxArgSum y, float it) {
  MaxArgSum r;
  if (y.m > x.m || (y.m == x.m && y.a < x.a)) { r.m = y.m; r.a = y.a; } else { r.m = x.m; r.a = x.a; }
  const float fx = x.m == -INFINITY ? 0.f : expf((x.m - r.m) * it);
  const float fy = y.m == -INFINITY ? 0.f : expf((y.m - r.m) * it);
  r.s = x.s * fx + y.s * fy;
  return r;
}

// One CTA per token row: merge the per-vocab-tile partials, then subtract
// the log-sum-exp from the scaled logits already stored in logsoftmax.
__global__ void lm_reduce_kernel(const float* __restrict__ pmax, const int* __restrict__ parg,
                                 const float* __restrict__ psum, int tiles, long long M, long long V,
                                 float it, int* tok, float* zmax, float* ls) {
  __shared__ MaxArgSum sh[32];
  __shared__ float lse_sh;
  const long long j = blockIdx.x;
  MaxArgSum acc{-INFINITY, INT_MAX, 0.f};
  for (int t = threadIdx.x; t < tiles; t += blockDim.x) {
    const size_t o = (size_t)t * M + j;
    acc = combine(acc, MaxArgSum{pmax[o], parg[o], psum[o]}, it);
  }
  for (int off = 16; off > 0; off >>= 1) {
    MaxArgSum o{__shfl_xor_sync(0xffffffffu, acc.m, off), __shfl_xor_sync(0xffffffffu, acc.a, off),
                __shfl_xor_sync(0xffffffffu, acc.s, off)};
    acc = combine(acc, o, it);
  }
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (lane == 0) sh[warp] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    MaxArgSum r = sh[0];
    for (int w = 1; w < (int)(blockDim.x >> 5); ++w) r = combine(r, sh[w], it);
    tok[j] = r.a;
    if (zmax) zmax[j] = r.m;
    lse_sh = r.m * it + logf(r.s);
  }
  __syncthreads();
  if (ls) {
    const float lse = lse_sh;
    float* row = ls + j * V;
    for (long long v = threadIdx.x; v < V; v += blockDim.x) row[v] -= lse;
  }
}

}  // namespace

cudaError_t launch_rope_table(double theta, int hd, long long max_pos, float* c, float* s,
                              cudaStream_t st) {
  const long long n = max_pos * (hd / 2);
  if (n == 0) return cudaSuccess;
  const int blocks = (int)std::min<long long>((n + 255) / 256, 4096);
  rope_table_kernel<<<blocks, 256, 0, st>>>(theta, hd, max_pos, c, s);
  return cudaGetLastError();
}

cudaError_t launch_rmsnorm(const void* x, int x_is_f32, const void* w, void* y, int dtype, long long rows,
                           int d, float eps, cudaStream_t s) {
  if (rows == 0) return cudaSuccess;
  if (dtype == HDF_BF16) {
    if (x_is_f32)
      rmsnorm_kernel<float, __nv_bfloat16><<<(unsigned)rows, 256, 0, s>>>(
          (const float*)x, (const __nv_bfloat16*)w, (__nv_bfloat16*)y, d, eps);
    else
      rmsnorm_bf16_vec_kernel<<<(unsigned)rows, 128, 0, s>>>((const __nv_bfloat16*)x,
                                                             (const __nv_bfloat16*)w, (__nv_bfloat16*)y, d, eps);
  } else {
    rmsnorm_kernel<float, float><<<(unsigned)rows, 256, 0, s>>>((const float*)x, (const float*)w, (float*)y,
                                                                d, eps);
  }
  return cudaGetLastError();
}

cudaError_t launch_embed_norm(const void* embed, const void* mask_vec, const int* anchor, const void* norm_w,
                              float* h, void* x, int dtype, int batch, int block, int d, int vocab, float eps,
                              cudaStream_t s) {
  const int rows = batch * block;
  if (rows == 0) return cudaSuccess;
  if (dtype == HDF_BF16)
    embed_norm_kernel<__nv_bfloat16><<<rows, 256, 0, s>>>(
        (const __nv_bfloat16*)embed, (const __nv_bfloat16*)mask_vec, anchor, (const __nv_bfloat16*)norm_w, h,
        (__nv_bfloat16*)x, block, d, vocab, eps);
  else
    embed_norm_kernel<float><<<rows, 256, 0, s>>>((const float*)embed, (const float*)mask_vec, anchor,
                                                  (const float*)norm_w, h, (float*)x, block, d, vocab, eps);
  return cudaGetLastError();
}

cudaError_t launch_accept(const int* draft, long long ds, const int* target, long long ts, int batch, int nd,
                          int* accept, cudaStream_t s) {
  if (batch == 0) return cudaSuccess;
  accept_kernel<<<(batch + 127) / 128, 128, 0, s>>>(draft, ds, target, ts, batch, nd, accept);
  return cudaGetLastError();
}

cudaError_t launch_lm_reduce(const float* pmax, const int* parg, const float* psum, int tiles, long long M,
                             long long V, float it, int* tok, float* zmax, float* ls, cudaStream_t s) {
  if (M == 0) return cudaSuccess;
  lm_reduce_kernel<<<(unsigned)M, 256, 0, s>>>(pmax, parg, psum, tiles, M, V, it, tok, zmax, ls);
  return cudaGetLastError();
}

}  // namespace hdf
