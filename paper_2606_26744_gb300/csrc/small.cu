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

// Row RMSNorm, y = x / sqrt(mean(x^2) + eps) * w, one CTA of 256 threads
// per row.  Every thread loads its VPT 16-byte vectors of the row at once
// (all in flight), keeps them in registers across the reduction and writes
// y once: one read and one write of the row, no dependent load chains.
// XT is the input type (fp32 residual or T), T the output/weight type.
// With EMBED the row is [embed[anchor]; mask_vec x (B-1)] and is also
// written to the fp32 residual h.
template <typename XT, typename T, int VPT, bool EMBED>
__global__ void __launch_bounds__(256) rmsnorm_vec_kernel(const XT* __restrict__ x, const T* __restrict__ w,
                                                          T* __restrict__ y, int d, float eps,
                                                          const int* __restrict__ anchor,
                                                          const T* __restrict__ mask_vec, float* __restrict__ h,
                                                          int block, int vocab) {
  constexpr int XV = 16 / sizeof(XT);  // input elements per 16-byte vector
  __shared__ float sh[32];
  pdl_launch_dependents();
  pdl_wait();
  const long long r = blockIdx.x;
  const XT* xr = x + r * d;
  if (EMBED) {  // x is the embedding table here
    const int i = (int)(r / block), k = (int)(r - (long long)i * block);
    const int tokid = min(max(__ldg(anchor + i), 0), vocab - 1);  // ids outside [0, V) are clamped
    xr = k == 0 ? x + (long long)tokid * d : reinterpret_cast<const XT*>(mask_vec);
  }
  const int nv = d / XV;
  float v[VPT][XV];
  float ss = 0.f;
#pragma unroll
  for (int k = 0; k < VPT; ++k) {
    const int i = threadIdx.x + k * 256;
    uint4 raw = make_uint4(0, 0, 0, 0);
    if (i < nv) raw = ld_nc16(xr + (size_t)i * XV);
    V16<XT>::unpack(raw, v[k]);
#pragma unroll
    for (int e = 0; e < XV; ++e) ss = fmaf(v[k][e], v[k][e], ss);
  }
  const float inv = rsqrtf(block_sum(ss, sh) / (float)d + eps);
#pragma unroll
  for (int k = 0; k < VPT; ++k) {
    const int i = threadIdx.x + k * 256;
    if (i >= nv) continue;
    if (EMBED) {
#pragma unroll
      for (int e = 0; e < XV; e += 4)
        *reinterpret_cast<float4*>(h + r * d + (size_t)i * XV + e) =
            make_float4(v[k][e], v[k][e + 1], v[k][e + 2], v[k][e + 3]);
    }
    float g[XV];
    if constexpr (sizeof(T) == 2 && XV == 8) {
      V16<T>::unpack(ld_nc16(w + (size_t)i * 8), g);
    } else if constexpr (sizeof(T) == 2 && XV == 4) {
      const uint2 raw = __ldg(reinterpret_cast<const uint2*>(w + (size_t)i * 4));
      g[0] = bf16lo(raw.x); g[1] = bf16hi(raw.x); g[2] = bf16lo(raw.y); g[3] = bf16hi(raw.y);
    } else {
      V16<float>::unpack(ld_nc16(w + (size_t)i * 4), g);
    }
    float o[XV];
#pragma unroll
    for (int e = 0; e < XV; ++e) o[e] = v[k][e] * inv * g[e];
    T* yr = y + r * d + (size_t)i * XV;
    if constexpr (sizeof(T) == 2 && XV == 8) {
      *reinterpret_cast<uint4*>(yr) = V16<T>::pack(o);
    } else if constexpr (sizeof(T) == 2 && XV == 4) {
      *reinterpret_cast<uint2*>(yr) = make_uint2(pack_bf16x2(o[0], o[1]), pack_bf16x2(o[2], o[3]));
    } else {
      *reinterpret_cast<uint4*>(yr) = V16<float>::pack(o);
    }
  }
}

template <typename XT, typename T, bool EMBED>
cudaError_t launch_norm_t(const void* x, const void* w, void* y, long long rows, int d, float eps,
                          const int* anchor, const void* mask_vec, float* h, int block, int vocab,
                          cudaStream_t s) {
  constexpr int XV = 16 / sizeof(XT);
  const int vpt = (d / XV + 255) / 256;
  const dim3 grid((unsigned)rows);
#define HDF_NORM_LAUNCH(N)                                                                              \
  launch_kernel(rmsnorm_vec_kernel<XT, T, N, EMBED>, grid, dim3(256), 0, s, 1u, (const XT*)x, (const T*)w, \
                (T*)y, d, eps, anchor, (const T*)mask_vec, h, block, vocab)
  if (vpt <= 1) return HDF_NORM_LAUNCH(1);
  if (vpt <= 2) return HDF_NORM_LAUNCH(2);
  if (vpt <= 4) return HDF_NORM_LAUNCH(4);
  if (vpt <= 8) return HDF_NORM_LAUNCH(8);
  if (vpt <= 16) return HDF_NORM_LAUNCH(16);
#undef HDF_NORM_LAUNCH
  return cudaErrorInvalidValue;
}

// Accepted-prefix length (Sec. 3.4): n_i = the number of leading draft
// tokens equal to the target's.  A CTA stages the rows of ACC_ROWS sequences
// of both inputs in shared memory with coalesced loads (consecutive threads,
// consecutive entries), then each thread scans its own row there.
constexpr int ACC_ROWS = 128;
__global__ void __launch_bounds__(ACC_ROWS) accept_kernel(const int* __restrict__ draft, long long ds,
                                                          const int* __restrict__ target, long long ts, int batch,
                                                          int nd, int* __restrict__ accept) {
  extern __shared__ int acc_sm[];  // [2][ACC_ROWS][nd]
  pdl_launch_dependents();
  pdl_wait();
  const long long r0 = (long long)blockIdx.x * ACC_ROWS;
  const int rows = (int)min((long long)ACC_ROWS, (long long)batch - r0);
  int* sd = acc_sm;
  int* st = acc_sm + ACC_ROWS * nd;
  const int total = rows * nd;
  if (nd > 0) {
    // entry e = r * nd + k, advanced by ACC_ROWS entries a step without a division
    const int rstep = ACC_ROWS / nd, kstep = ACC_ROWS - rstep * nd;
    int r = threadIdx.x / nd, k = threadIdx.x - r * nd;
    for (int base = threadIdx.x; base < total; base += 8 * ACC_ROWS) {
      int vd[8], vt[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {  // eight pairs of loads in flight before any store
        if (base + u * ACC_ROWS < total) {
          vd[u] = __ldcs(draft + (r0 + r) * ds + k);
          vt[u] = __ldcs(target + (r0 + r) * ts + k);
        }
        r += rstep;
        k += kstep;
        if (k >= nd) {
          k -= nd;
          ++r;
        }
      }
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int e = base + u * ACC_ROWS;
        if (e < total) {
          sd[e] = vd[u];
          st[e] = vt[u];
        }
      }
    }
  }
  __syncthreads();
  const int i = threadIdx.x;
  if (i >= rows) return;
  int n = 0;
  while (n < nd && sd[i * nd + n] == st[i * nd + n]) ++n;
  accept[r0 + i] = n;
}

// Cache length update after an append: len[b] += n_b (n_b = cu[b+1] - cu[b]),
// limited to the capacity; a count that is negative or passes the capacity
// is recorded (the append kernel skipped those rows).
__global__ void cache_advance_kernel(int* __restrict__ len, const int* __restrict__ cu, int batch, long long cap,
                                     int* status) {
  pdl_launch_dependents();
  pdl_wait();  // every layer's append has read len
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= batch) return;
  const long long n = (long long)cu[b + 1] - cu[b];
  long long t = (long long)len[b] + n;
  if (n < 0 || t > cap) {
    record_device_error(status);
    t = t < 0 ? 0 : (t > cap ? cap : t);
    if (n < 0) t = len[b];
  }
  len[b] = (int)t;
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

// CTA (j, c): merge token row j's per-vocabulary-tile partials (every CTA of
// the row in the same order, so all get the same bits), then subtract the
// log-sum-exp from vocabulary chunk c of the scaled logits already stored in
// logsoftmax (16-byte accesses when rows are 16-byte multiples).  Chunk 0
// writes the row's token and maximal logit.
constexpr long long kLsChunk = 8192;  // vocabulary entries normalised per CTA

__global__ void lm_reduce_kernel(const float* __restrict__ pmax, const int* __restrict__ parg,
                                 const float* __restrict__ psum, int tiles, long long M, long long V,
                                 float it, int* tok, float* zmax, float* ls) {
  __shared__ MaxArgSum sh[32];
  __shared__ float lse_sh;
  pdl_launch_dependents();
  pdl_wait();
  const long long j = blockIdx.x;
  const long long chunk = blockIdx.y;
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
    if (chunk == 0) {
      tok[j] = r.a;
      if (zmax) zmax[j] = r.m;
    }
    lse_sh = r.m * it + logf(r.s);
  }
  __syncthreads();
  if (ls) {
    const float lse = lse_sh;
    float* row = ls + j * V;
    const long long v0 = chunk * kLsChunk, v1 = min(V, v0 + kLsChunk);
    if ((V & 3) == 0) {
      float4* r4 = reinterpret_cast<float4*>(row);
      for (long long q = v0 / 4 + threadIdx.x; q < v1 / 4; q += blockDim.x) {
        float4 x = r4[q];
        x.x -= lse;
        x.y -= lse;
        x.z -= lse;
        x.w -= lse;
        r4[q] = x;
      }
    } else {
      for (long long v = v0 + threadIdx.x; v < v1; v += blockDim.x) row[v] -= lse;
    }
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
      return launch_norm_t<float, __nv_bfloat16, false>(x, w, y, rows, d, eps, nullptr, nullptr, nullptr, 1, 1, s);
    return launch_norm_t<__nv_bfloat16, __nv_bfloat16, false>(x, w, y, rows, d, eps, nullptr, nullptr, nullptr, 1,
                                                              1, s);
  }
  return launch_norm_t<float, float, false>(x, w, y, rows, d, eps, nullptr, nullptr, nullptr, 1, 1, s);
}

cudaError_t launch_embed_norm(const void* embed, const void* mask_vec, const int* anchor, const void* norm_w,
                              float* h, void* x, int dtype, int batch, int block, int d, int vocab, float eps,
                              cudaStream_t s) {
  const int rows = batch * block;
  if (rows == 0) return cudaSuccess;
  if (dtype == HDF_BF16)
    return launch_norm_t<__nv_bfloat16, __nv_bfloat16, true>(embed, norm_w, x, rows, d, eps, anchor, mask_vec, h,
                                                             block, vocab, s);
  return launch_norm_t<float, float, true>(embed, norm_w, x, rows, d, eps, anchor, mask_vec, h, block, vocab, s);
}

cudaError_t launch_accept(const int* draft, long long ds, const int* target, long long ts, int batch, int nd,
                          int* accept, cudaStream_t s) {
  if (batch == 0) return cudaSuccess;
  return launch_kernel(accept_kernel, dim3((unsigned)((batch + ACC_ROWS - 1) / ACC_ROWS)), dim3(ACC_ROWS),
                       (size_t)2 * ACC_ROWS * nd * sizeof(int), s, 1u, draft, ds, target, ts, batch, nd, accept);
}

cudaError_t launch_cache_advance(int* len, const int* cu, int batch, long long cap, int* status, cudaStream_t s) {
  if (batch == 0) return cudaSuccess;
  return launch_kernel(cache_advance_kernel, dim3((batch + 127) / 128), dim3(128), 0, s, 1u, len, cu, batch, cap,
                       status);
}

cudaError_t launch_lm_reduce(const float* pmax, const int* parg, const float* psum, int tiles, long long M,
                             long long V, float it, int* tok, float* zmax, float* ls, cudaStream_t s) {
  if (M == 0) return cudaSuccess;
  const unsigned chunks = ls ? (unsigned)((V + kLsChunk - 1) / kLsChunk) : 1u;
  return launch_kernel(lm_reduce_kernel, dim3((unsigned)M, chunks), dim3(256), 0, s, 1u, pmax, parg, psum, tiles, M,
                       V, it, tok, zmax, ls);
}

}  // namespace hdf
