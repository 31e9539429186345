// Temperature-1 block verification by speculative sampling (the T = 1 rows
// of Tables 2 and 3 of the HyperDFlash paper; the standard rule it relies on):
//   accept draft slot k when u / 2^32 < p(x) / q(x) (one IEEE fp32 division),
//   stop at the first rejection; draw the next token from norm(max(0, p - q))
//   at the rejected slot (from p there if that residual is empty), or from p
//   at the bonus slot when every draft is accepted.
// The draw is exact integer arithmetic: weights floor(w * 2^40), threshold
// floor(r * R / 2^32), the token is the first whose prefix sum exceeds it.
// One CTA of 32 warps per sequence; warp w owns a contiguous slice of the
// vocabulary, read 32 entries at a time (coalesced); warp sums are scanned in
// warp order, and the warp whose slice holds the threshold finds the token
// with a warp prefix scan.  Everything after the fp32 subtraction is integer,
// so the result is independent of scheduling.
#include "common.cuh"
#include "kernels.h"

namespace hdf {
namespace {

constexpr int VS_WARPS = 32;

__device__ __forceinline__ unsigned long long weight_fixed(float w) {
  // w in [0, 1]: w * 2^40 is exact in double; truncation is floor for w >= 0
  return w > 0.f ? (unsigned long long)((double)w * 1099511627776.0) : 0ull;
}

// weight of entry v of the chosen distribution: max(0, p - q) or p
__device__ __forceinline__ unsigned long long entry_weight(const float* __restrict__ p, const float* __restrict__ q,
                                                           long long v) {
  const float w = q ? fmaxf(__fsub_rn(p[v], q[v]), 0.f) : p[v];
  return weight_fixed(w);
}

__device__ __forceinline__ unsigned long long warp_sum_u64(unsigned long long x) {
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  return x;
}

__global__ void __launch_bounds__(32 * VS_WARPS) accept_sample_kernel(
    const float* __restrict__ pt, const float* __restrict__ qd, const int* __restrict__ draft, long long dstride,
    const unsigned* __restrict__ u, const unsigned* __restrict__ r, int nd, long long V, int* __restrict__ accept,
    int* __restrict__ next_tok) {
  __shared__ int n_s;
  __shared__ unsigned long long wsum[VS_WARPS], wexcl[VS_WARPS];
  __shared__ unsigned long long total_s, thr_s;
  pdl_launch_dependents();
  pdl_wait();
  const long long i = blockIdx.x;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    int n = 0;
    while (n < nd) {
      const int x = draft[i * dstride + n];
      if (x < 0 || x >= V) break;  // an id outside the vocabulary is rejected
      const float pv = pt[((i * (nd + 1)) + n) * V + x];
      const float qv = qd[((i * nd) + n) * V + x];
      const float ratio = __fdiv_rn(pv, qv);  // p/0 = inf: accept; 0/0 = nan: reject
      if ((double)u[i * nd + n] * 2.3283064365386963e-10 < (double)ratio) ++n;
      else break;
    }
    n_s = n;
    accept[i] = n;
  }
  __syncthreads();
  const int n = n_s;
  const float* p = pt + ((i * (nd + 1)) + n) * V;
  const float* q = n < nd ? qd + ((i * nd) + n) * V : nullptr;
  const long long C = ((V + VS_WARPS - 1) / VS_WARPS + 31) / 32 * 32;  // slice per warp, multiple of 32
  const long long c0 = warp * C, c1 = min(V, c0 + C);
  for (int attempt = 0; attempt < 2; ++attempt) {
    unsigned long long s = 0;
    for (long long v = c0 + lane; v < c1; v += 32) s += entry_weight(p, q, v);
    s = warp_sum_u64(s);
    if (lane == 0) wsum[warp] = s;
    __syncthreads();
    if (tid == 0) {
      unsigned long long run = 0;
      for (int w = 0; w < VS_WARPS; ++w) {
        wexcl[w] = run;
        run += wsum[w];
      }
      total_s = run;
      // floor(r * R / 2^32), exact: R < 2^63
      const unsigned long long rr = r[i];
      thr_s = (run >> 32) * rr + (((run & 0xffffffffull) * rr) >> 32);
    }
    __syncthreads();
    if (total_s != 0 || q == nullptr) break;
    q = nullptr;  // empty residual: draw from p at the rejected slot
    __syncthreads();
  }
  const unsigned long long total = total_s, thr = thr_s;
  if (total == 0) {
    if (tid == 0) next_tok[i] = -1;
    return;
  }
  // the warp whose slice holds the threshold
  if (wsum[warp] != 0 && wexcl[warp] <= thr && thr < wexcl[warp] + wsum[warp]) {
    unsigned long long base = wexcl[warp];
    for (long long v0 = c0; v0 < c1; v0 += 32) {
      const long long v = v0 + lane;
      const unsigned long long w = v < c1 ? entry_weight(p, q, v) : 0ull;
      unsigned long long incl = w;  // inclusive prefix within these 32 entries
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const unsigned long long t = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += t;
      }
      const unsigned hit = __ballot_sync(0xffffffffu, base + incl > thr);
      if (hit) {
        if (lane == __ffs(hit) - 1) next_tok[i] = (int)v;
        break;
      }
      base += __shfl_sync(0xffffffffu, incl, 31);
    }
  }
}

}  // namespace

cudaError_t launch_accept_sample(const float* p, const float* q, const int* draft, long long dstride,
                                 const unsigned* u, const unsigned* r, int batch, int nd, long long V, int* accept,
                                 int* next_tok, cudaStream_t s) {
  if (batch == 0) return cudaSuccess;
  return launch_kernel(accept_sample_kernel, dim3((unsigned)batch), dim3(32 * VS_WARPS), 0, s, 1u, p, q, draft,
                       dstride, u, r, nd, V, accept, next_tok);
}

}  // namespace hdf
