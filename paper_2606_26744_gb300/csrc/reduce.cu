// Inherited HC-Gate reducer, Eq. 1 of the HyperDFlash paper (Sec. 2.2).
//
// Per token t with pre-collapse residual H_t in R^{m x d}:
//   r      = (mean(vec(H_t)^2) + eps)^(-1/2)
//   alpha_j= sigmoid(s * r * (W_f vec H_t)_j + b_j) + offset
//   y_t    = sum_j alpha_j * H^_tj   (H^ = H, or the per-path RMSNorm)
//
// Memory-bound streaming design.  A persistent CTA owns a fixed slice of
// every token: thread i handles the 16-byte vectors v = i, i + nt, ... of the
// d axis for all m paths, so the weighted sum over paths is in-thread and the
// W_f columns a thread needs never change (kept in shared memory when they
// fit, else read through L1).  G tokens are processed together so each W_f
// load feeds G tokens.  Phase 1 streams H from HBM (L1 no-allocate) and
// accumulates the m gate dots and m per-path sums of squares; a transposed
// warp butterfly plus one shared-memory pass reduces them across the CTA.
// Phase 2 re-reads the same G tokens (now L2-resident: one HBM pass) and
// writes y once.
#include "common.cuh"
#include "kernels.h"

namespace hdf {
namespace {

constexpr int next_pow2(int x) { return x <= 1 ? 1 : 2 * next_pow2((x + 1) / 2); }

template <typename T, int M, int G, bool WF_SMEM>
__global__ void __launch_bounds__(512) gated_reduce_kernel(const ReduceArgs a, int vpt) {
  constexpr int VEC = V16<T>::N;
  constexpr int NV = next_pow2(G * 2 * M);  // reduced values per token group (padded)
  static_assert(NV <= 32, "reduction values must fit one warp");
  extern __shared__ __align__(16) uint8_t dyn_smem[];
  __shared__ float red[32][NV];
  __shared__ float fin[NV];

  const int tid = threadIdx.x, nt = blockDim.x, lane = tid & 31, warp = tid >> 5;
  const int nwarps = nt >> 5;
  const int d = a.d, md = M * d, nvec = d / VEC;
  const long long n = a.n_tokens;
  const T* __restrict__ H = reinterpret_cast<const T*>(a.H);
  const T* Wf = reinterpret_cast<const T*>(a.Wf);

  const bool use_gate = a.alpha_override == nullptr;
  if (WF_SMEM && use_gate) {
    const uint4* src = reinterpret_cast<const uint4*>(a.Wf);
    uint4* dst = reinterpret_cast<uint4*>(dyn_smem);
    const int n16 = (M * md * (int)sizeof(T)) / 16;
    for (int i = tid; i < n16; i += nt) dst[i] = __ldg(src + i);
    __syncthreads();
    Wf = reinterpret_cast<const T*>(dyn_smem);
  }

  const long long ngroups = (n + G - 1) / G;
  for (long long grp = blockIdx.x; grp < ngroups; grp += gridDim.x) {
    const long long t0 = grp * G;
    float acc[NV];
#pragma unroll
    for (int i = 0; i < NV; ++i) acc[i] = 0.f;

    // ---- phase 1: gate dot products and per-path sums of squares
    for (int k = 0; k < vpt; ++k) {
      const int v = tid + k * nt;
      if (v < nvec) {
#pragma unroll
        for (int p = 0; p < M; ++p) {
          float h[G][VEC];
#pragma unroll
          for (int g = 0; g < G; ++g) {
            uint4 raw = make_uint4(0, 0, 0, 0);
            if (t0 + g < n) raw = ld_stream16(H + (t0 + g) * md + p * d + v * VEC);
            V16<T>::unpack(raw, h[g]);
          }
#pragma unroll
          for (int j = 0; j < M; ++j) {
            if (!use_gate) break;
            const T* wp = Wf + (size_t)j * md + p * d + v * VEC;
            uint4 wr = WF_SMEM ? *reinterpret_cast<const uint4*>(wp) : ld_nc16(wp);
            float w[VEC];
            V16<T>::unpack(wr, w);
#pragma unroll
            for (int g = 0; g < G; ++g)
#pragma unroll
              for (int e = 0; e < VEC; ++e) acc[g * 2 * M + j] = fmaf(w[e], h[g][e], acc[g * 2 * M + j]);
          }
#pragma unroll
          for (int g = 0; g < G; ++g)
#pragma unroll
            for (int e = 0; e < VEC; ++e)
              acc[g * 2 * M + M + p] = fmaf(h[g][e], h[g][e], acc[g * 2 * M + M + p]);
        }
      }
    }

    // ---- CTA reduction: transposed butterfly leaves value (lane % NV) on each lane
#pragma unroll
    for (int o = NV / 2; o >= 1; o >>= 1) {
      const bool upper = (lane & o) != 0;
#pragma unroll
      for (int i = 0; i < o; ++i) {
        const float send = upper ? acc[i] : acc[i + o];
        const float keep = upper ? acc[i + o] : acc[i];
        acc[i] = keep + __shfl_xor_sync(0xffffffffu, send, o);
      }
    }
#pragma unroll
    for (int o = NV; o < 32; o <<= 1) acc[0] += __shfl_xor_sync(0xffffffffu, acc[0], o);
    if (lane < NV) red[warp][lane] = acc[0];
    __syncthreads();
    if (tid < NV) {
      float s = 0.f;
      for (int w = 0; w < nwarps; ++w) s += red[w][tid];
      fin[tid] = s;
    }
    __syncthreads();

    // ---- gates
    float alpha[G][M], rp[G][M];
#pragma unroll
    for (int g = 0; g < G; ++g) {
      const float* f = fin + g * 2 * M;
      float ss = 0.f;
#pragma unroll
      for (int p = 0; p < M; ++p) ss += f[M + p];
      const float r = rsqrtf(ss / (float)md + a.rms_eps);
      const long long t = t0 + g;
#pragma unroll
      for (int j = 0; j < M; ++j) {
        if (a.alpha_override) {
          alpha[g][j] = (t < n) ? a.alpha_override[t * M + j] : 0.f;
        } else {
          const float logit = a.gate_scale * r * f[j] + a.b[j];
          alpha[g][j] = 1.0f / (1.0f + expf(-logit)) + a.gate_offset;
        }
        rp[g][j] = a.path_norm_w ? rsqrtf(f[M + j] / (float)d + a.path_norm_eps) : 1.f;
      }
      if (a.alpha_out && tid < M && t < n) {
#pragma unroll
        for (int j = 0; j < M; ++j)
          if (j == tid) a.alpha_out[t * M + j] = alpha[g][j];
      }
    }

    // ---- phase 2: weighted sum over paths (H re-read from L2), one store
    const T* pnw = reinterpret_cast<const T*>(a.path_norm_w);
    T* y = reinterpret_cast<T*>(a.y);
    for (int k = 0; k < vpt; ++k) {
      const int v = tid + k * nt;
      if (v >= nvec) continue;
#pragma unroll
      for (int g = 0; g < G; ++g) {
        const long long t = t0 + g;
        if (t >= n) continue;
        float out[VEC];
#pragma unroll
        for (int e = 0; e < VEC; ++e) out[e] = 0.f;
#pragma unroll
        for (int p = 0; p < M; ++p) {
          float h[VEC];
          V16<T>::unpack(ld_nc16(H + t * md + p * d + v * VEC), h);
          if (pnw) {
            float gm[VEC];
            V16<T>::unpack(ld_nc16(pnw + p * d + v * VEC), gm);
            const float s = alpha[g][p] * rp[g][p];
#pragma unroll
            for (int e = 0; e < VEC; ++e) out[e] = fmaf(s * gm[e], h[e], out[e]);
          } else {
#pragma unroll
            for (int e = 0; e < VEC; ++e) out[e] = fmaf(alpha[g][p], h[e], out[e]);
          }
        }
        *reinterpret_cast<uint4*>(y + t * d + v * VEC) = V16<T>::pack(out);
      }
    }
  }
}

template <typename T, int M>
cudaError_t launch_m(const ReduceArgs& a, cudaStream_t s) {
  constexpr int G = (M >= 8) ? 2 : 4;
  constexpr int VEC = V16<T>::N;
  const int nvec = a.d / VEC;
  const int vpt = (nvec + 511) / 512;
  int nt = (nvec + vpt - 1) / vpt;
  nt = ((nt + 31) / 32) * 32;
  const size_t wf_bytes = (size_t)M * M * a.d * sizeof(T);
  const bool wf_smem = wf_bytes <= 160 * 1024 && a.alpha_override == nullptr;
  int dev = 0, sms = 0, per_sm = 0;
  cudaError_t e;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
  const long long ngroups = (a.n_tokens + G - 1) / G;
  if (wf_smem) {
    auto k = gated_reduce_kernel<T, M, G, true>;
    if ((e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)wf_bytes)) != cudaSuccess)
      return e;
    if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k, nt, wf_bytes)) != cudaSuccess) return e;
    if (per_sm < 1) per_sm = 1;
    const long long grid = std::min<long long>(ngroups, (long long)per_sm * sms);
    k<<<(unsigned)grid, nt, wf_bytes, s>>>(a, vpt);
  } else {
    auto k = gated_reduce_kernel<T, M, G, false>;
    if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k, nt, 0)) != cudaSuccess) return e;
    if (per_sm < 1) per_sm = 1;
    const long long grid = std::min<long long>(ngroups, (long long)per_sm * sms);
    k<<<(unsigned)grid, nt, 0, s>>>(a, vpt);
  }
  return cudaGetLastError();
}

template <typename T>
cudaError_t launch_t(const ReduceArgs& a, cudaStream_t s) {
  switch (a.m) {
    case 1: return launch_m<T, 1>(a, s);
    case 2: return launch_m<T, 2>(a, s);
    case 3: return launch_m<T, 3>(a, s);
    case 4: return launch_m<T, 4>(a, s);
    case 8: return launch_m<T, 8>(a, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

cudaError_t launch_gated_reduce(const ReduceArgs& a, int dtype, cudaStream_t s) {
  if (a.n_tokens == 0) return cudaSuccess;
  return dtype == HDF_BF16 ? launch_t<__nv_bfloat16>(a, s) : launch_t<float>(a, s);
}

}  // namespace hdf
