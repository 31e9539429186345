// Gradient of the gated residual reducer (Eq. 1, Sec. 2.2 of the HyperDFlash
// paper) with respect to its trainable gate parameters W_f [m, m*d] and
// b [m], the 65K parameters of Table 1, for L = sum_t dy_t . y_t with the
// target's residual H held fixed (no per-path norm, no gate override):
//   r_t   = (mean(vec H_t ^2) + eps)^-1/2,  g_tj = s r_t (W_f vec H_t)_j + b_j
//   dg_tj = (dy_t . H_tj) sigmoid'(g_tj),  sigmoid'(g) = sigmoid(g) sigmoid(-g)
//   db_j  = sum_t dg_tj,   dW_f[j] = sum_t (s r_t dg_tj) vec(H_t)
// Three passes, every sum in a fixed order (bitwise reproducible):
//   1. gate: a CTA takes RB_TOK tokens at a time; thread k owns the 16-byte
//      vectors k, k + 256, ... of vec H_t and accumulates sum x^2, the m gate
//      dots (each W_f vector load serves RB_TOK tokens) and the m dots
//      dy_t . H_tj; warp butterflies, then the warps in order; one thread per
//      path writes dg_tj and u_tj = s r_t dg_tj.
//   2. weight gradient: CTA (slice, split) owns 256 x VEC columns of W_f and a
//      contiguous token range; each thread keeps m x VEC fp32 sums over its
//      tokens in token order (and the CTAs of slice 0 the db sums) and writes
//      them to the split's partial.  The CTA streams its 4 KB slice of 16
//      tokens at a time (and their u rows) through a 3-deep cp.async ring in
//      shared memory, one CTA per SM: 128 KB of H in flight per SM.
//   3. finalize: the partials are added in split order.
// HBM-bound: H is read twice (passes 1 and 2), dy once.
#include <algorithm>

#include "common.cuh"
#include "kernels.h"

namespace hdf {
namespace {

constexpr int RB_THREADS = 256;
constexpr int RB_TOK = 4;  // tokens per CTA iteration in pass 1
constexpr int RB_WARPS = RB_THREADS / 32;

template <typename T, int M>
__global__ void __launch_bounds__(RB_THREADS) reduce_bwd_gate_kernel(const ReduceBwdArgs a) {
  pdl_launch_dependents();
  pdl_wait();
  constexpr int VEC = V16<T>::N;
  const int d = a.d;
  const int vpp = d / VEC;  // vectors per path
  const int nv = M * vpp;   // vectors per token
  const long long md = (long long)M * d;
  const T* H = reinterpret_cast<const T*>(a.H);
  const T* dy = reinterpret_cast<const T*>(a.dy);
  const T* Wf = reinterpret_cast<const T*>(a.Wf);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  constexpr int NV = 2 * M + 1;  // sum x^2, M gate dots, M dy dots
  __shared__ float red[RB_WARPS][RB_TOK][NV];
  const float inv_md = 1.0f / (float)md;

  for (long long t0 = (long long)blockIdx.x * RB_TOK; t0 < a.n_tokens; t0 += (long long)gridDim.x * RB_TOK) {
    const int nt = (int)min((long long)RB_TOK, a.n_tokens - t0);
    float acc[RB_TOK][NV];
#pragma unroll
    for (int i = 0; i < RB_TOK; ++i)
#pragma unroll
      for (int k = 0; k < NV; ++k) acc[i][k] = 0.f;
    for (int v = tid; v < nv; v += RB_THREADS) {
      const int p = v / vpp;
      const int off = (v - p * vpp) * VEC;
      float w[M][VEC];
#pragma unroll
      for (int j = 0; j < M; ++j) V16<T>::unpack(ld_nc16(Wf + (long long)j * md + (long long)v * VEC), w[j]);
#pragma unroll
      for (int i = 0; i < RB_TOK; ++i) {
        if (i < nt) {
          const long long t = t0 + i;
          float x[VEC], g[VEC];
          V16<T>::unpack(ld_nc16(H + t * md + (long long)v * VEC), x);
          V16<T>::unpack(ld_nc16(dy + t * d + off), g);
          float ss = 0.f, da = 0.f;
#pragma unroll
          for (int e = 0; e < VEC; ++e) {
            ss += x[e] * x[e];
            da += g[e] * x[e];
          }
          acc[i][0] += ss;
#pragma unroll
          for (int j = 0; j < M; ++j) {
            float q = 0.f;
#pragma unroll
            for (int e = 0; e < VEC; ++e) q += w[j][e] * x[e];
            acc[i][1 + j] += q;
            if (j == p) acc[i][1 + M + j] += da;
          }
        }
      }
    }
#pragma unroll
    for (int i = 0; i < RB_TOK; ++i)
#pragma unroll
      for (int k = 0; k < NV; ++k) {
        const float s = warp_sum(acc[i][k]);
        if (lane == 0) red[warp][i][k] = s;
      }
    __syncthreads();
    if (tid < RB_TOK * M) {
      const int i = tid / M, j = tid - i * M;
      if (i < nt) {
        float ss = 0.f, q = 0.f, al = 0.f;
        for (int w = 0; w < RB_WARPS; ++w) {  // the warps in order
          ss += red[w][i][0];
          q += red[w][i][1 + j];
          al += red[w][i][1 + M + j];
        }
        const float r = rsqrtf(ss * inv_md + a.rms_eps);
        const float g = a.gate_scale * r * q + a.b[j];
        // sigmoid'(g) = sigmoid(g) sigmoid(-g): no cancellation where sigmoid(g) rounds to 1
        const float dg = al * sigmoidf_(g) * sigmoidf_(-g);
        const long long t = t0 + i;
        a.dg[t * M + j] = dg;
        a.u[t * M + j] = a.gate_scale * r * dg;
      }
    }
    __syncthreads();  // red[] is reused by the next tokens
  }
}

constexpr int WG_TOK = 16;    // tokens per ring stage
constexpr int WG_STAGES = 3;  // ring depth
constexpr int wg_stage_bytes(int m) { return WG_TOK * RB_THREADS * 16 + WG_TOK * 8 * 4; }  // H slice + u rows
constexpr size_t wg_smem(int m) { return (size_t)WG_STAGES * wg_stage_bytes(m); }

__device__ __forceinline__ void cp_async16(void* dst, const void* src, bool pred) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.u32 p, %2, 0;\n @p cp.async.cg.shared.global [%0], [%1], 16;\n}\n" ::"r"(
          smem_u32(dst)),
      "l"(src), "r"((uint32_t)pred)
      : "memory");
}
__device__ __forceinline__ void cp_async4(void* dst, const void* src, bool pred) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.u32 p, %2, 0;\n @p cp.async.ca.shared.global [%0], [%1], 4;\n}\n" ::"r"(
          smem_u32(dst)),
      "l"(src), "r"((uint32_t)pred)
      : "memory");
}

template <typename T, int M>
__global__ void __launch_bounds__(RB_THREADS, 1) reduce_bwd_wgrad_kernel(const ReduceBwdArgs a, long long tok_per) {
  extern __shared__ __align__(16) uint8_t wg_smem_raw[];
  pdl_launch_dependents();
  pdl_wait();
  constexpr int VEC = V16<T>::N;
  constexpr int SB = wg_stage_bytes(M);
  const long long md = (long long)M * a.d;
  const T* H = reinterpret_cast<const T*>(a.H);
  const int tid = threadIdx.x;
  const int split = blockIdx.y;
  const long long t0 = (long long)split * tok_per;
  const long long t1 = min(a.n_tokens, t0 + tok_per);
  const long long c = ((long long)blockIdx.x * RB_THREADS + tid) * VEC;  // first column of this thread
  const bool active = c < md;
  const bool db_thread = blockIdx.x == 0 && tid < M;
  const long long ntok = t1 > t0 ? t1 - t0 : 0;
  const long long nstage = (ntok + WG_TOK - 1) / WG_TOK;
  // stage g: tokens t0 + g*WG_TOK .. ; this thread copies its 16 bytes of
  // every token, threads 0 .. WG_TOK*M-1 one u entry each
  auto issue = [&](long long g) {
    uint8_t* st = wg_smem_raw + (g % WG_STAGES) * SB;
    const long long tb = t0 + g * WG_TOK;
#pragma unroll
    for (int i = 0; i < WG_TOK; ++i) {
      const long long t = tb + i;
      cp_async16(st + (i * RB_THREADS + tid) * 16, H + (t < t1 ? t : t0) * md + (active ? c : 0), active && t < t1);
    }
    if (tid < WG_TOK * M) {
      const int i = tid / M, j = tid - i * M;
      const long long t = tb + i;
      cp_async4(st + WG_TOK * RB_THREADS * 16 + (i * 8 + j) * 4, a.u + (t < t1 ? t : t0) * M + j, t < t1);
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  };
  float acc[M][VEC];
#pragma unroll
  for (int j = 0; j < M; ++j)
#pragma unroll
    for (int e = 0; e < VEC; ++e) acc[j][e] = 0.f;
  float dbs = 0.f;
  for (long long g = 0; g < WG_STAGES - 1; ++g) {
    if (g < nstage) issue(g);
    else asm volatile("cp.async.commit_group;" ::: "memory");
  }
  for (long long g = 0; g < nstage; ++g) {
    if (g + WG_STAGES - 1 < nstage) issue(g + WG_STAGES - 1);
    else asm volatile("cp.async.commit_group;" ::: "memory");
    asm volatile("cp.async.wait_group %0;" ::"n"(WG_STAGES - 1) : "memory");  // stage g has landed (this thread's copies)
    __syncthreads();                                                           // ... and every thread's
    const uint8_t* st = wg_smem_raw + (g % WG_STAGES) * SB;
    const float* us = reinterpret_cast<const float*>(st + WG_TOK * RB_THREADS * 16);
    const long long tb = t0 + g * WG_TOK;
    const int nt = (int)min((long long)WG_TOK, t1 - tb);
    if (active) {
#pragma unroll 4
      for (int i = 0; i < WG_TOK; ++i) {
        if (i < nt) {  // tokens in order
          float x[VEC];
          V16<T>::unpack(*reinterpret_cast<const uint4*>(st + (i * RB_THREADS + tid) * 16), x);
#pragma unroll
          for (int j = 0; j < M; ++j) {
            const float u = us[i * 8 + j];
#pragma unroll
            for (int e = 0; e < VEC; ++e) acc[j][e] += u * x[e];
          }
        }
      }
    }
    if (db_thread)
      for (int i = 0; i < nt; ++i) dbs += __ldg(a.dg + (tb + i) * M + tid);
    __syncthreads();  // the stage is read before it is refilled
  }
  asm volatile("cp.async.wait_all;" ::: "memory");
  if (active) {
#pragma unroll
    for (int j = 0; j < M; ++j) {
      float* dst = a.part + ((long long)split * M + j) * md + c;
#pragma unroll
      for (int e = 0; e < VEC; e += 4)
        *reinterpret_cast<float4*>(dst + e) = make_float4(acc[j][e], acc[j][e + 1], acc[j][e + 2], acc[j][e + 3]);
    }
  }
  if (db_thread) a.dbpart[(long long)split * M + tid] = dbs;
}

__global__ void reduce_bwd_finalize_kernel(const ReduceBwdArgs a, int n_split) {
  pdl_launch_dependents();
  pdl_wait();
  const long long n = (long long)a.m * a.m * a.d;  // entries of W_f
  for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n + a.m;
       i += (long long)gridDim.x * blockDim.x) {
    if (i < n) {
      float s = 0.f;
      for (int k = 0; k < n_split; ++k) s += a.part[(long long)k * n + i];  // splits in order
      a.dWf[i] = s;
    } else {
      const int j = (int)(i - n);
      float s = 0.f;
      for (int k = 0; k < n_split; ++k) s += a.dbpart[(long long)k * a.m + j];
      a.db[j] = s;
    }
  }
}

template <typename T, int M>
cudaError_t launch_m(const ReduceBwdArgs& a, const ReduceBwdPlan& p, cudaStream_t s) {
  cudaError_t e = launch_kernel(reduce_bwd_gate_kernel<T, M>, dim3((unsigned)p.gate_ctas), dim3(RB_THREADS), 0, s,
                                1u, a);
  if (e != cudaSuccess) return e;
  if ((e = ensure_smem_limit((const void*)reduce_bwd_wgrad_kernel<T, M>, wg_smem(M))) != cudaSuccess) return e;
  e = launch_kernel(reduce_bwd_wgrad_kernel<T, M>, dim3((unsigned)p.slices, (unsigned)p.splits), dim3(RB_THREADS),
                    wg_smem(M), s, 1u, a, p.tok_per);
  if (e != cudaSuccess) return e;
  const long long n = (long long)M * M * a.d + M;
  const unsigned blocks = (unsigned)std::min<long long>((n + 255) / 256, 4096);
  return launch_kernel(reduce_bwd_finalize_kernel, dim3(blocks), dim3(256), 0, s, 1u, a, p.splits);
}

template <typename T>
cudaError_t launch_t(const ReduceBwdArgs& a, const ReduceBwdPlan& p, cudaStream_t s) {
  switch (a.m) {
    case 1: return launch_m<T, 1>(a, p, s);
    case 2: return launch_m<T, 2>(a, p, s);
    case 3: return launch_m<T, 3>(a, p, s);
    case 4: return launch_m<T, 4>(a, p, s);
    case 8: return launch_m<T, 8>(a, p, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

ReduceBwdPlan reduce_bwd_plan(long long n_tokens, int m, int d, int dtype, int n_sm) {
  ReduceBwdPlan p;
  if (n_tokens <= 0) return p;  // nothing to launch
  const int vec = dtype == HDF_BF16 ? 8 : 4;
  const long long md = (long long)m * d;
  p.slices = (int)((md + (long long)RB_THREADS * vec - 1) / ((long long)RB_THREADS * vec));
  const long long want = std::max(1LL, (long long)n_sm / p.slices);  // one CTA per SM
  p.splits = (int)std::max(1LL, std::min({want, 1024LL, n_tokens}));
  p.tok_per = (n_tokens + p.splits - 1) / p.splits;
  p.splits = (int)std::max(1LL, (n_tokens + p.tok_per - 1) / p.tok_per);  // no empty split
  p.gate_ctas = (int)std::max(1LL, std::min(2LL * n_sm, (n_tokens + RB_TOK - 1) / RB_TOK));
  return p;
}

cudaError_t launch_gated_reduce_backward(const ReduceBwdArgs& a, int dtype, const ReduceBwdPlan& p, cudaStream_t s) {
  return dtype == HDF_BF16 ? launch_t<__nv_bfloat16>(a, p, s) : launch_t<float>(a, p, s);
}

}  // namespace hdf
