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
  __shared__ float red[16][NV];  // one row per warp (at most 512 threads)
  __shared__ float fin[NV];
  __shared__ float bias_s[M];
  __shared__ float gate_s[G][M][2];  // alpha and the path-norm factor of each (token, path)

  const int tid = threadIdx.x, nt = blockDim.x, lane = tid & 31, warp = tid >> 5;
  pdl_launch_dependents();
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
  if (tid < M && use_gate) bias_s[tid] = a.b[tid];
  __syncthreads();
  pdl_wait();  // H, y and alpha_override may belong to the kernels before

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

    // ---- gates: one thread per (token, path), shared through shared memory
    if (tid < G * M) {
      const int g = tid / M, j = tid - g * M;
      const float* f = fin + g * 2 * M;
      float ss = 0.f;
#pragma unroll
      for (int p = 0; p < M; ++p) ss += f[M + p];
      const float r = rsqrtf(ss / (float)md + a.rms_eps);
      const long long t = t0 + g;
      float al;
      if (a.alpha_override) {
        al = (t < n) ? a.alpha_override[t * M + j] : 0.f;
      } else {
        const float logit = a.gate_scale * r * f[j] + bias_s[j];
        al = 1.0f / (1.0f + expf(-logit)) + a.gate_offset;
      }
      gate_s[g][j][0] = al;
      gate_s[g][j][1] = a.path_norm_w ? rsqrtf(f[M + j] / (float)d + a.path_norm_eps) : 1.f;
      if (a.alpha_out && t < n) a.alpha_out[t * M + j] = al;
    }
    __syncthreads();
    float alpha[G][M], rp[G][M];
#pragma unroll
    for (int g = 0; g < G; ++g)
#pragma unroll
      for (int j = 0; j < M; ++j) {
        alpha[g][j] = gate_s[g][j][0];
        rp[g][j] = gate_s[g][j][1];
      }

    // ---- phase 2: weighted sum over paths (H re-read from L2), one store;
    // every load of a vector's G x M values is issued before its stores
    const T* pnw = reinterpret_cast<const T*>(a.path_norm_w);
    T* __restrict__ y = reinterpret_cast<T*>(a.y);
    for (int k = 0; k < vpt; ++k) {
      const int v = tid + k * nt;
      if (v >= nvec) continue;
      uint4 raw[G][M];
#pragma unroll
      for (int g = 0; g < G; ++g)
#pragma unroll
        for (int p = 0; p < M; ++p)
          raw[g][p] = t0 + g < n ? ld_nc16(H + (t0 + g) * md + p * d + v * VEC) : make_uint4(0, 0, 0, 0);
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
          V16<T>::unpack(raw[g][p], h);
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
  // W_f in shared memory up to 160 KB: larger (m = 4, d = 7168) would leave
  // one CTA per SM, which costs more than reading W_f through L1 / L2
  const bool wf_smem = wf_bytes <= 160 * 1024 && a.alpha_override == nullptr;
  int dev = 0, sms = 0, per_sm = 0;
  cudaError_t e;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
  const long long ngroups = (a.n_tokens + G - 1) / G;
  auto go = [&](auto k, size_t smem) -> cudaError_t {
    cudaError_t e2;
    if (smem > 48 * 1024 && (e2 = ensure_smem_limit((const void*)k, smem)) != cudaSuccess) return e2;
    if ((e2 = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k, nt, smem)) != cudaSuccess) return e2;
    if (per_sm < 1) per_sm = 1;
    const long long grid = std::min<long long>(ngroups, (long long)per_sm * sms);
    return launch_kernel(k, dim3((unsigned)grid), dim3(nt), smem, s, 1u, a, vpt);
  };
  if (wf_smem) return go(gated_reduce_kernel<T, M, G, true>, wf_bytes);
  return go(gated_reduce_kernel<T, M, G, false>, 0);
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

// ===========================================================================
// bf16 cluster path (the hot path of Eq. 1).
//
// A cluster of 8 CTAs shares every token: CTA rank c owns elements
// [c*E, (c+1)*E) of each of the m paths (E = d/8), so its slice of W_f
// (m x m*E, 28 KB at d = 7168) stays in shared memory for the whole run.
// Tokens move in batches of RB (8, or 4 when the slice is wide).  The warps
// of a CTA have fixed roles and meet only at mbarriers:
//   producer warp   one TMA box per path per batch from the 3-D view
//                   {64 elements, tokens, 128-byte chunks} of H, which lands
//                   as [chunk][token][64 elements] rows of 128 bytes with the
//                   128-byte swizzle, so ldmatrix reads any 8 of them without
//                   bank conflicts
//   NGW gate warps  split every batch's tiles; each warp owns the same tiles
//                   in every batch, so its W_f fragments and shared-memory
//                   offsets stay in registers.  On the tensor cores
//                   (mma.sync m16n8k16) the 16 rows of a tile are (token,
//                   k-range) pairs, RB tokens x KR = 16/RB k-ranges of 16
//                   elements; the 8 columns are (gate, k-range) pairs of W_f,
//                   and only the blocks whose k-ranges agree are kept.  The
//                   sums of squares come from the same A fragments on the
//                   FP32 pipe.  Pairs of gate warps combine their partials and
//                   send them to every rank with st.async, which completes the
//                   receiver's exchange mbarrier on bytes.  A slot goes back
//                   to the producer as soon as the gate warps are done with
//                   it, so most of the ring is always loading.
//   alpha warp      sums every batch's partials over all senders in a fixed
//                   order (the same on every rank, so every rank gets the same
//                   alpha) and publishes alpha for the batch
//   NWW weighted    take whole batches in turn and write the y slice, reading
//   warps           H again: the batch was streamed a few microseconds before
//                   and is still in L2
// Gate warps run at most LA batches ahead of the alpha warp, which bounds how
// far any rank can run ahead in the exchange.  H comes from HBM once, W_f once
// per CTA.
namespace {

constexpr int RC = 8;              // CTAs per cluster
constexpr int NGW = 8;             // gate warps
constexpr int GGRP = 2;            // gate warps whose partials are combined before they are sent
constexpr int MAXT = 8;            // tiles per gate warp and batch (fragments held in registers)
constexpr int NWW = 6;             // weighted warps
constexpr int NAB = NWW + 2;       // published alpha buffers
constexpr int NTHR = 32 * (2 + NGW + NWW);  // + producer warp + alpha warp
constexpr int LA = 4;              // gate warps run at most this many batches ahead
constexpr int NXCH = 2 * LA + 2;   // exchange buffers (a rank sends batch j only after this rank used j - 2*LA)
constexpr int NSRC = RC * NGW / GGRP;  // partial senders per batch: (rank, gate warp group), one per lane

struct RedGeo {
  int E;       // elements per path in a CTA slice
  int rb;      // tokens per batch (4 or 8)
  int ws;      // W_f slice row stride (bytes): m*E*2 + 16
  int box;     // bytes of one path's box: E * rb * 2
  int preg;    // path region stride in a slot: box rounded up to 1024 bytes
  int slot;    // bytes per batch slot: m * preg
  int ring;    // batch slots
  int xbuf;    // bytes of one exchange buffer: NSRC rows of rb * (m+1) partials
  long long nbatch;
};

__device__ __forceinline__ void ldsm_x2(uint32_t addr, uint32_t& r0, uint32_t& r1) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.shared.b16 {%0,%1}, [%2];" : "=r"(r0), "=r"(r1) : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void mma16816(float* d, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* map, int x, int y, int z, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
      "l"((uint64_t)map), "r"(x), "r"(y), "r"(z), "r"(bar)
      : "memory");
}

// acc.{x,y} += (bf16 pair of w)^2, both halves at once
__device__ __forceinline__ void sq_acc2(unsigned long long& acc, uint32_t w) {
  const unsigned long long v = ((unsigned long long)(w & 0xffff0000u) << 32) | (unsigned long long)(w << 16);
  asm("fma.rn.f32x2 %0, %1, %1, %0;" : "+l"(acc) : "l"(v));
}
__device__ __forceinline__ float sum2(unsigned long long v) {
  return __uint_as_float((uint32_t)v) + __uint_as_float((uint32_t)(v >> 32));
}

// k-step (16 elements of a path slice) that k-range kr of tile step s covers.
// Every k-step is covered once.  The order keeps the W_f rows one B fragment
// reads, (gate, k-range) pairs, in distinct bank groups: k-ranges that share
// an 8-column tile sit 2 k-steps (64 bytes) apart.
template <int KR>
__device__ __forceinline__ int kstep_of(int s, int kr) {
  if (KR == 4) return 4 * s + ((kr & 1) << 1) + (kr >> 1);  // 0, 2, 1, 3
  return 4 * (s >> 1) + 2 * kr + (s & 1);                   // KR == 2
}

template <int M, int RB>
__global__ void __launch_bounds__(NTHR, 1)
    gated_reduce_cluster_kernel(const ReduceArgs a, const RedGeo geo, const __grid_constant__ CUtensorMap hmap) {
  constexpr int KR = 16 / RB;          // k-ranges per tile
  constexpr int NCOL = M * KR;         // (gate, k-range) columns
  constexpr int NT = (NCOL + 7) / 8;   // 8-column tiles (2 only for m = 4, RB = 4)
  constexpr int NV = M + 1;            // partials per token: m gate dots, sum of squares
  constexpr int XV = RB * NV;          // partials per sender
  constexpr int U = M == 1 ? 8 : 16 / M;  // weighted outputs per lane and round (8-16 loads in flight)
  constexpr uint32_t kXchBytes = NSRC * XV * 4;  // one batch's partials from all senders
  static_assert(RB * M <= 32, "one lane per alpha");
  static_assert(NSRC == 32 && XV % 4 == 0 && XV <= 64, "one sender per lane; rows are read as float4");

  extern __shared__ __align__(128) uint8_t sm[];
  __shared__ __align__(8) uint64_t full_bar[16];
  __shared__ __align__(8) uint64_t empty_bar[16];
  __shared__ __align__(8) uint64_t xfull[NXCH];
  __shared__ __align__(8) uint64_t xdone[NXCH];        // the alpha warp has read an exchange buffer
  __shared__ __align__(8) uint64_t alpha_ready[NAB];
  __shared__ __align__(8) uint64_t alpha_free[NAB];
  __shared__ float red[NGW][16][NV];    // per gate warp: tile row (token, k-range) x partial
  __shared__ float alpha_s[NAB][RB][M];
  __shared__ float bias_s[M];
  __shared__ volatile int abort_flag;
  __shared__ volatile int group_abort[NGW / GGRP];  // written and read by one gate warp group only

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  pdl_launch_dependents();
  const uint32_t rank = cluster_rank(), cid = cluster_id_x(), ncl = n_clusters_x();
  const int d = a.d, E = geo.E, e0 = (int)rank * E;
  const long long n = a.n_tokens;
  uint8_t* wsm = sm;  // [M gates][ws bytes]
  // TMA destinations start on a 128-byte boundary: the ring starts on the
  // next 1024-byte boundary after the W_f slice (the launch adds the slack)
  const uint32_t sm0 = smem_u32(sm);
  uint8_t* ring = sm + (((sm0 + M * geo.ws + 1023u) & ~1023u) - sm0);  // [ring][m paths][chunk][RB][128 B]
  float* xch = reinterpret_cast<float*>(ring + (size_t)geo.ring * geo.slot);  // [NXCH][NSRC][XV]

  // W_f slice: row j = gate j, flat slice index k = p*E + e
  {
    const int per_row16 = M * E / 8;
    const __nv_bfloat16* Wf = reinterpret_cast<const __nv_bfloat16*>(a.Wf);
    for (int i = tid; i < M * per_row16; i += blockDim.x) {
      const int j = i / per_row16, r = i - j * per_row16;
      const int p = (r * 8) / E, e = r * 8 - p * E;
      *reinterpret_cast<uint4*>(wsm + j * geo.ws + r * 16) =
          __ldg(reinterpret_cast<const uint4*>(Wf + (size_t)j * M * d + (size_t)p * d + e0 + e));
    }
  }
  const long long nl = geo.nbatch > (long long)cid ? (geo.nbatch - cid + ncl - 1) / ncl : 0;
  if (tid < M) bias_s[tid] = a.b[tid];
  if (tid == 0) {
    for (int s = 0; s < geo.ring; ++s) {
      mbar_init(smem_u32(&full_bar[s]), 1);
      mbar_init(smem_u32(&empty_bar[s]), NGW);
    }
    // exchange barriers complete on bytes: every rank's st.async signals them
    for (int b = 0; b < NXCH; ++b) {
      mbar_init(smem_u32(&xfull[b]), 1);
      mbar_init(smem_u32(&xdone[b]), 1);
    }
    for (int b = 0; b < NAB; ++b) {
      mbar_init(smem_u32(&alpha_ready[b]), 1);
      mbar_init(smem_u32(&alpha_free[b]), 1);
    }
    abort_flag = 0;
    for (int gg = 0; gg < NGW / GGRP; ++gg) group_abort[gg] = 0;
    fence_mbar_init();
    for (int b = 0; b < NXCH && b < nl; ++b) mbar_arrive_expect_tx(smem_u32(&xfull[b]), kXchBytes);
  }
  __syncthreads();
  cluster_sync_all();  // every rank's barriers exist (and are armed) before anyone signals them remotely
  pdl_wait();          // H and y may belong to the kernels before

  // a wait that every lane of the warp takes; false (for the whole warp) on
  // time-out or when another warp has given up
  auto warp_wait = [&](uint32_t bar, uint32_t parity, bool cluster_scope) -> bool {
    bool got = cluster_scope ? mbar_wait_cluster(bar, parity, a.status) : mbar_wait(bar, parity, a.status);
    got = __all_sync(0xffffffffu, got) && !__any_sync(0xffffffffu, abort_flag != 0);
    if (!got && lane == 0) abort_flag = 1;
    return got;
  };
  auto arrive = [&](uint64_t* bar) {
    if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
  };

  if (warp == 0) {
    if (lane == 0) {  // ---------------------------------------------- producer
      prefetch_tmap(&hmap);
      long long issued = 0;
      for (long long i = 0; i < nl && !abort_flag; ++i) {
        const int slot = (int)(i % geo.ring);
        const uint32_t ph = (uint32_t)((i / geo.ring) & 1);
        if (!mbar_wait(smem_u32(&empty_bar[slot]), ph ^ 1, a.status)) { abort_flag = 1; break; }
        const long long t0 = ((long long)cid + i * ncl) * RB;
        const uint32_t fb = smem_u32(&full_bar[slot]);
        mbar_arrive_expect_tx(fb, (uint32_t)(M * geo.box));
        const uint32_t dst = smem_u32(ring + (size_t)slot * geo.slot);
#pragma unroll
        for (int p = 0; p < M; ++p)
          tma_load_3d(dst + p * geo.preg, &hmap, 0, (int)t0, (p * d + e0) / 64, fb);
        issued = i + 1;
      }
      // no copy may still be landing when the CTA exits: wait for the last
      // batch of every slot (already complete on the normal path)
      for (long long i = issued > geo.ring ? issued - geo.ring : 0; i < issued; ++i)
        if (!mbar_wait(smem_u32(&full_bar[i % geo.ring]), (uint32_t)((i / geo.ring) & 1), a.status)) break;
    }
    __syncwarp();
  } else if (warp <= NGW) {
    // ------------------------------------------------------------ gate warps
    const int gw = warp - 1, grp = gw / GGRP;
    const int g = lane >> 2, q = lane & 3;
    // Tiles go in units of two tile steps (s = 2*sp, 2*sp+1) of one path;
    // unit u = gw + NGW*k belongs to this warp, its tiles are k = 2*(u/NGW) + c.
    const int SP = E / (16 * KR);  // tile steps per path
    const int NP = (SP + 1) / 2;   // units per path
    // A operand, ldmatrix.x4: lane -> matrix mi (rows 0-7 / 8-15, k 0-7 / 8-15), row R
    const int mi = lane >> 3, Ra = (lane & 7) + 8 * (mi & 1), khA = mi >> 1;
    const int tA = Ra % RB, krA = Ra / RB;
    // B operand (W_f), ldmatrix.x2 / x4: lane -> column n = (gate, k-range), k half
    const int nB = 8 * (lane >> 4) + (lane & 7), khB = (lane >> 3) & 1;
    const int jB = nB < NCOL ? nB % M : 0, krB = nB < NCOL ? nB / M : 0;
    uint32_t aoff[MAXT], bf[MAXT][NT][2];
    unsigned valid = 0;  // the same for every lane
    {
      int p = 0, sp = gw;
      while (sp >= NP) { sp -= NP; ++p; }
#pragma unroll
      for (int k = 0; k < MAXT; ++k) {
        if (k > 0 && (k & 1) == 0) {
          sp += NGW;
          while (sp >= NP) { sp -= NP; ++p; }
        }
        const int s = 2 * sp + (k & 1);
        const bool v = p < M && s < SP;
        if (v) valid |= 1u << k;
        const int pv = v ? p : 0, sv = v ? s : 0;
        const int ka = kstep_of<KR>(sv, krA);
        const int row = (ka >> 2) * RB + tA, un = ((ka & 3) << 1) | khA;
        aoff[k] = pv * geo.preg + row * 128 + ((un ^ (row & 7)) << 4);
        const uint32_t baddr =
            smem_u32(wsm + jB * geo.ws + khB * 16) + (uint32_t)(pv * E + 16 * kstep_of<KR>(sv, krB)) * 2;
        if (NT == 2)
          ldsm_x4(baddr, bf[k][0][0], bf[k][0][1], bf[k][NT - 1][0], bf[k][NT - 1][1]);
        else
          ldsm_x2(baddr, bf[k][0][0], bf[k][0][1]);
      }
    }
    // the warps of a group meet at a named barrier (ids 1..NGW/GGRP)
    auto group_sync = [&]() {
      if (GGRP > 1) asm volatile("bar.sync %0, %1;" ::"r"(1 + grp), "r"(32 * GGRP) : "memory");
    };
    for (long long i = 0; i < nl; ++i) {
      bool w_ok = true;
      if (i >= LA) {  // credit: the alpha warp has read the partials of batch i - LA
        const long long c = i - LA;
        w_ok = warp_wait(smem_u32(&xdone[c % NXCH]), (uint32_t)((c / NXCH) & 1), false);
      }
      const int slot = (int)(i % geo.ring);
      if (w_ok) w_ok = warp_wait(smem_u32(&full_bar[slot]), (uint32_t)((i / geo.ring) & 1), false);
      if (GGRP > 1) {
        // one decision for the whole group: a flag written before the
        // barrier, read after it, never by anyone else
        if (!w_ok && lane == 0) group_abort[grp] = 1;
        group_sync();
        if (group_abort[grp]) break;
      } else if (!w_ok) {
        break;
      }
      const uint32_t sbase = smem_u32(ring + (size_t)slot * geo.slot);
      uint32_t av[MAXT][4];
#pragma unroll
      for (int k = 0; k < MAXT; ++k)
        if (valid >> k & 1) ldsm_x4(sbase + aoff[k], av[k][0], av[k][1], av[k][2], av[k][3]);
      __syncwarp();  // this warp is done with the slot
      arrive(&empty_bar[slot]);
      float dg[2][NT][4];  // chain: tile parity
      unsigned long long sl[2] = {0ull, 0ull}, sh[2] = {0ull, 0ull};  // sums of squares, rows g and g + 8
#pragma unroll
      for (int c = 0; c < 2; ++c)
#pragma unroll
        for (int t = 0; t < NT; ++t) dg[c][t][0] = dg[c][t][1] = dg[c][t][2] = dg[c][t][3] = 0.f;
#pragma unroll
      for (int k = 0; k < MAXT; ++k) {
        if (valid >> k & 1) {
#pragma unroll
          for (int t = 0; t < NT; ++t) mma16816(dg[k & 1][t], av[k], bf[k][t][0], bf[k][t][1]);
          sq_acc2(sl[k & 1], av[k][0]);
          sq_acc2(sl[k & 1], av[k][2]);
          sq_acc2(sh[k & 1], av[k][1]);
          sq_acc2(sh[k & 1], av[k][3]);
        }
      }
      // keep the blocks whose k-ranges agree, and the sums of squares
#pragma unroll
      for (int t = 0; t < NT; ++t) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int R = g + 8 * (e >> 1), ncol = 8 * t + 2 * q + (e & 1);
          if (ncol < NCOL && ncol / M == R / RB) red[gw][R][ncol % M] = dg[0][t][e] + dg[1][t][e];
        }
      }
      {
        float lo = sum2(sl[0]) + sum2(sl[1]), hi = sum2(sh[0]) + sum2(sh[1]);
        lo += __shfl_xor_sync(0xffffffffu, lo, 1);
        hi += __shfl_xor_sync(0xffffffffu, hi, 1);
        lo += __shfl_xor_sync(0xffffffffu, lo, 2);
        hi += __shfl_xor_sync(0xffffffffu, hi, 2);
        if (q == 0) {
          red[gw][g][M] = lo;
          red[gw][g + 8][M] = hi;
        }
      }
      __syncwarp();
      group_sync();  // the group's partials are complete
      // the group's first warp sends; red is rewritten only after the next
      // batch's group barrier, which that warp reaches after its sends
      for (int x = lane; x < XV && gw % GGRP == 0; x += 32) {
        const int tk = x / NV, k = x - tk * NV;
        float v = 0.f;
#pragma unroll
        for (int h = 0; h < GGRP; ++h)
#pragma unroll
          for (int kr = 0; kr < KR; ++kr) v += red[gw + h][kr * RB + tk][k];
        const int b = (int)(i % NXCH);
        const uint32_t lx = smem_u32(xch + ((size_t)b * NSRC + rank * (NGW / GGRP) + grp) * XV + x);
        const uint32_t lb = smem_u32(&xfull[b]);
#pragma unroll
        for (uint32_t r = 0; r < RC; ++r)
          asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.f32 [%0], %1, [%2];" ::"r"(
                           map_rank(lx, r)),
                       "f"(v), "r"(map_rank(lb, r))
                       : "memory");
      }
      __syncwarp();
    }
  } else if (warp == NGW + 1) {
    // ------------------------------------------------------------ alpha warp
    long long consumed = 0;
    bool ok = true;
    for (long long i = 0; i < nl; ++i) {
      consumed = i;
      const int b = (int)(i % NXCH);
      if (!warp_wait(smem_u32(&xfull[b]), (uint32_t)((i / NXCH) & 1), true)) {
        ok = false;
        break;
      }
      // buffer b is complete: arm it for batch i + NXCH (no rank sends that
      // batch before this warp has read batch i + 2)
      if (lane == 0 && i + NXCH < nl) mbar_arrive_expect_tx(smem_u32(&xfull[b]), kXchBytes);
      // lane L holds sender L's partials; a transposed butterfly sums them
      // over the 32 senders in a fixed order and leaves partial x on lane x
      // (and on lane x - 32 for x >= 32)
      constexpr int XP = XV <= 32 ? 32 : 64;  // padded
      float v[XP];
      const float4* row = reinterpret_cast<const float4*>(xch + ((size_t)b * NSRC + lane) * XV);
#pragma unroll
      for (int k = 0; k < XP / 4; ++k) {
        const float4 f = k < XV / 4 ? row[k] : make_float4(0.f, 0.f, 0.f, 0.f);
        v[4 * k] = f.x;
        v[4 * k + 1] = f.y;
        v[4 * k + 2] = f.z;
        v[4 * k + 3] = f.w;
      }
      __syncwarp();
      arrive(&xdone[b]);
#pragma unroll
      for (int h = 0; h < XP / 32; ++h) {
        float* w = v + 32 * h;
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) {
          const bool upper = (lane & o) != 0;
#pragma unroll
          for (int k = 0; k < o; ++k) {
            const float send = upper ? w[k] : w[k + o];
            const float keep = upper ? w[k + o] : w[k];
            w[k] = keep + __shfl_xor_sync(0xffffffffu, send, o);
          }
        }
      }
      const int tk = lane / M, j = lane - tk * M;
      const int xg = tk * NV + j, xs = tk * NV + M;
      const float g0 = __shfl_sync(0xffffffffu, v[0], xg & 31), s0 = __shfl_sync(0xffffffffu, v[0], xs & 31);
      float gl = g0, ssum = s0;
      if (XP == 64) {
        const float g1 = __shfl_sync(0xffffffffu, v[XP == 64 ? 32 : 0], xg & 31);
        const float s1 = __shfl_sync(0xffffffffu, v[XP == 64 ? 32 : 0], xs & 31);
        gl = xg >= 32 ? g1 : g0;
        ssum = xs >= 32 ? s1 : s0;
      }
      const int ab = (int)(i % NAB);
      if (i >= NAB && !warp_wait(smem_u32(&alpha_free[ab]), (uint32_t)(((i / NAB) - 1) & 1), false)) {
        ok = false;
        break;
      }
      const long long t0 = ((long long)cid + i * ncl) * RB;
      const int nv = (int)min((long long)RB, n - t0);
      if (lane < RB * M) {
        const float rr = rsqrtf(ssum / (float)(M * d) + a.rms_eps);
        const float al = 1.0f / (1.0f + expf(-(a.gate_scale * rr * gl + bias_s[j]))) + a.gate_offset;
        alpha_s[ab][tk][j] = al;
        if (a.alpha_out && rank == 0 && tk < nv) a.alpha_out[(t0 + tk) * M + j] = al;
      }
      __syncwarp();
      arrive(&alpha_ready[ab]);
    }
    if (!ok && lane == 0) {
      // abort: let the other ranks' partials already on their way land
      // before the cluster exits (one shared time limit for all of them)
      const unsigned long long t0 = globaltimer_ns();
      for (long long j = consumed; j < nl && j < consumed + NXCH; ++j) {
        const uint32_t bar = smem_u32(&xfull[j % NXCH]), par = (uint32_t)((j / NXCH) & 1);
        while (!mbar_try_wait_cluster(bar, par) && globaltimer_ns() - t0 < kWaitLimitNs) {
        }
      }
    }
  } else {
    // -------------------------------------------------------- weighted warps
    const int ww = warp - NGW - 2;
    const int nitems = (E / 64) * RB * 8;  // 16-byte output units of a batch's slice
    const __nv_bfloat16* H = reinterpret_cast<const __nv_bfloat16*>(a.H);
    __nv_bfloat16* y = reinterpret_cast<__nv_bfloat16*>(a.y);
    for (long long i = ww; i < nl; i += NWW) {
      const int ab = (int)(i % NAB);
      if (!warp_wait(smem_u32(&alpha_ready[ab]), (uint32_t)((i / NAB) & 1), false)) break;
      const long long t0 = ((long long)cid + i * ncl) * RB;
      const int nv = (int)min((long long)RB, n - t0);
      for (int w0 = lane; w0 < nitems; w0 += 32 * U) {
        // U outputs per lane, all U*m loads issued first (H comes from L2);
        // eight lanes cover one 128-byte run of a token row
        uint4 h[U][M];
        int tk[U], col[U];
#pragma unroll
        for (int r = 0; r < U; ++r) {
          const int wr = w0 + 32 * r;
          const int u = wr & 7, row = wr >> 3, z = row / RB;
          tk[r] = row - z * RB;
          col[r] = e0 + z * 64 + u * 8;
          const bool live = wr < nitems && tk[r] < nv;
          if (!live) tk[r] = -1;
#pragma unroll
          for (int p = 0; p < M; ++p)
            h[r][p] = live ? ld_stream16(H + ((t0 + tk[r]) * M + p) * d + col[r]) : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int r = 0; r < U; ++r) {
          if (tk[r] < 0) continue;
          float out[8];
#pragma unroll
          for (int e = 0; e < 8; ++e) out[e] = 0.f;
#pragma unroll
          for (int p = 0; p < M; ++p) {
            float x[8];
            V16<__nv_bfloat16>::unpack(h[r][p], x);
            const float al = alpha_s[ab][tk[r]][p];
#pragma unroll
            for (int e = 0; e < 8; ++e) out[e] = fmaf(al, x[e], out[e]);
          }
          *reinterpret_cast<uint4*>(y + (t0 + tk[r]) * d + col[r]) = V16<__nv_bfloat16>::pack(out);
        }
      }
      __syncwarp();  // alpha_s[ab] is free once every lane is past it
      arrive(&alpha_free[ab]);
    }
  }
  __syncthreads();
  cluster_sync_all();  // no rank still writes into this CTA's shared memory
}

bool cluster_geometry(const ReduceArgs& a, int dtype, RedGeo* geo, size_t* smem) {
  if (dtype != HDF_BF16 || a.alpha_override || a.path_norm_w) return false;
  if (a.n_tokens <= 0 || a.n_tokens > (1ll << 31) - 64) return false;  // TMA coordinates are 32-bit
  if (!(a.m == 1 || a.m == 2 || a.m == 4) || a.d % (RC * 64)) return false;
  geo->E = a.d / RC;
  if (geo->E / 64 > 256) return false;  // TMA box dimension limit

  geo->ws = a.m * geo->E * 2 + 16;
  const size_t budget = 219 * 1024;
  // batch size: the one that keeps more bytes loading (ring - 1 slots), 8 on a tie
  long long best = -1;
  for (int rb = 8; rb >= 4; rb /= 2) {
    // the gate warps' tiles must fit their registers: m * units per path <= NGW * MAXT / 2
    if (a.m * ((geo->E / (16 * (16 / rb)) + 1) / 2) > NGW * MAXT / 2) continue;
    RedGeo g = *geo;
    g.rb = rb;
    g.box = g.E * rb * 2;
    g.preg = (g.box + 1023) & ~1023;
    g.slot = a.m * g.preg;
    g.xbuf = NSRC * rb * (a.m + 1) * 4;
    const size_t fixed = (size_t)a.m * g.ws + (size_t)NXCH * g.xbuf + 1024;  // + alignment slack of the ring
    if (fixed >= budget) continue;
    g.ring = (int)std::min<long long>(16, (long long)((budget - fixed) / g.slot));
    const long long in_flight = (long long)(g.ring - 1) * g.slot;
    if (g.ring >= 3 && in_flight > best) {
      best = in_flight;
      *geo = g;
      *smem = fixed + (size_t)g.ring * g.slot;
    }
  }
  if (best < 0) return false;
  geo->nbatch = (a.n_tokens + geo->rb - 1) / geo->rb;
  return true;
}

template <int M, int RB>
cudaError_t launch_cluster_mr(const ReduceArgs& a, const RedGeo& geo, size_t smem, const CUtensorMap* hmap,
                              cudaStream_t s) {
  auto k = gated_reduce_cluster_kernel<M, RB>;
  cudaError_t e;
  int max_clusters = 0;
  if ((e = ensure_smem_limit((const void*)k, smem)) != cudaSuccess) return e;
  if ((e = max_active_clusters((const void*)k, NTHR, smem, RC, &max_clusters)) != cudaSuccess) return e;
  if (max_clusters < 1) return cudaErrorInvalidConfiguration;
  const long long ncl = std::min<long long>(max_clusters, geo.nbatch);
  return launch_kernel(k, dim3((unsigned)(ncl * RC)), dim3(NTHR), smem, s, (unsigned)RC, a, geo, *hmap);
}

template <int M>
cudaError_t launch_cluster_m(const ReduceArgs& a, const RedGeo& geo, size_t smem, const CUtensorMap* hmap,
                             cudaStream_t s) {
  return geo.rb == 8 ? launch_cluster_mr<M, 8>(a, geo, smem, hmap, s) : launch_cluster_mr<M, 4>(a, geo, smem, hmap, s);
}

}  // namespace

bool reduce_cluster_box(const ReduceArgs& a, int dtype, unsigned box[3]) {
  RedGeo geo;
  size_t smem;
  if (!cluster_geometry(a, dtype, &geo, &smem)) return false;
  box[0] = 64;
  box[1] = (unsigned)geo.rb;
  box[2] = (unsigned)(geo.E / 64);
  return true;
}

cudaError_t launch_gated_reduce_cluster(const ReduceArgs& a, const CUtensorMap* hmap, cudaStream_t s) {
  RedGeo geo;
  size_t smem;
  if (!cluster_geometry(a, HDF_BF16, &geo, &smem)) return cudaErrorInvalidValue;
  switch (a.m) {
    case 1: return launch_cluster_m<1>(a, geo, smem, hmap, s);
    case 2: return launch_cluster_m<2>(a, geo, smem, hmap, s);
    case 4: return launch_cluster_m<4>(a, geo, smem, hmap, s);
    default: return cudaErrorInvalidValue;
  }
}

// ===========================================================================
// bf16 tile path (persistent, warp-specialised).
//
// A cluster of S CTAs (S = 4, or 8 when the slices would not fit) walks
// tiles of T = 32 (or 16, for wide slices) consecutive tokens; CTA rank c
// owns elements [c*E, (c+1)*E) of each of the m paths (E = d/S), so its W_f
// slice (m x m*E) stays in shared memory; it arrives by m*m bulk copies on
// one mbarrier, in flight beside the first boxes of H.  Roles, meeting only
// at mbarriers:
//   producer warp   streams pass 1 of every tile from HBM into a 128 KB ring:
//                   one TMA box per stage from the 3-D view {64 elements,
//                   tokens, 128-byte chunks} of H, C chunks (C * 128
//                   contiguous bytes, C = 4 or 8) of T tokens, landing as
//                   planes [T tokens][64 elements] with the 128-byte
//                   swizzle; it never waits on the gates, so HBM streaming
//                   continues across tiles
//   8 gate warps    (row tile of 16 tokens) x (box phase 0..3): the m gate
//                   dots on mma.sync m16n8k16 (tokens are the rows, the W_f
//                   slice is B) and the sums of squares from the same A
//                   fragments; the four phases of a row tile are added in
//                   phase order and sent, [16 tokens][m + 1] partials, to
//                   every rank with st.async, which completes the receiver's
//                   exchange mbarrier on bytes
//   alpha warp      on every rank: waits for all senders of a tile, sums each
//                   token's partials over the ranks in rank order (so every
//                   rank gets the same alpha, Eq. 1) and publishes alpha
//   8 weighted      y = sum_j alpha_j H_j for the CTA's slice of the tile,
//   warps           reading H again from L2 (streamed microseconds before)
//                   with 16 loads in flight per lane, one store per output
// Gate warps run at most TP_LA tiles ahead of their own alpha warp, which
// bounds how far any rank runs ahead in the exchange (TP_NX buffers).  H comes
// from HBM once, W_f once per CTA.  Every wait is time-limited.
namespace {

constexpr int TP_RING = 128 * 1024;        // ring bytes
constexpr int TP_MAXST = 16;               // ring slots at most (16-token tiles)
constexpr int TP_NGW = 8;                  // gate warps: (sub, box phase 0..3)
constexpr int TP_NPH = TP_NGW / 2;         // box phases
// Box j of tile i is stage g = i*NB + j of the ring, slot g % NST, and is
// read by the two gate warps of phase j % 4.  With NB and NST multiples of 4
// (the tile geometry requires the first), slot g % NST only ever holds boxes
// of phase g % 4, and the box a gate warp waits for comes NST stages after
// one it read itself: no waiter is more than one fill ahead of a slot's
// barrier (an mbarrier parity wait tells adjacent phases apart only).
constexpr int TP_NWW = 8;                  // weighted warps
constexpr int TP_THR = 32 * (2 + TP_NGW + TP_NWW);
constexpr int TP_LA = 1;                   // gate warps run at most this many tiles ahead of the alpha warp
constexpr int TP_NX = 2 * TP_LA + 2;       // exchange buffers
constexpr int TP_NAB = 3;                  // alpha buffers
constexpr int TP_PS = 8;                   // floats per token in an exchange row (m + 1 <= 5 used)
constexpr int TP_U = 4;                    // weighted outputs per lane and round

struct TileGeo {
  int s;     // CTAs per cluster (4 or 8): the d split
  int t;     // tokens per tile (16 or 32)
  int ec;    // elements per path in a CTA slice (multiple of 64)
  int nkb;   // 128-byte chunks per path slice
  int c;     // 128-byte chunks per token in a box (4 or 8)
  int ngrp;  // boxes per path slice: ngrp - 1 of c chunks, then one of tail chunks
  int tail;  // chunks in the last box of a path slice (1..c)
  int wrow;  // row stride (elements) of the W_f slice in shared memory
  long long ntiles;
};
struct TileMaps {
  CUtensorMap main;  // box {64, T, c}
  CUtensorMap tail;  // box {64, T, tail}
};

__device__ __forceinline__ void st_async_v4(uint32_t addr, float4 v, uint32_t bar) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.f32 [%0], {%1,%2,%3,%4}, [%5];" ::"r"(addr),
               "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w), "r"(bar)
               : "memory");
}

// contiguous global -> shared copy completing on an mbarrier (16-byte aligned
// addresses, size a multiple of 16)
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
               "l"(src), "r"(bytes), "r"(bar)
               : "memory");
}

// one tile's partials from all senders
constexpr int tp_xbytes(int S, int T) { return S * T * TP_PS * 4; }
constexpr size_t tp_smem(int S, int T, int m, int wrow) {
  return 1024 + (size_t)TP_RING + (size_t)tp_xbytes(S, T) * TP_NX + (size_t)TP_NPH * 32 * TP_PS * 4 +
         (size_t)TP_NAB * T * 16 + (size_t)m * wrow * 2;
}

// T tokens per tile: 32 (two 16-row tiles; the two gate warps of a phase
// take one each) or 16 (one row tile; the two gate warps of a phase take the
// even and the odd planes of every box).
template <int M, int S, int T, int TP_C>
__global__ void __launch_bounds__(TP_THR, 1) gated_reduce_tile_kernel(const ReduceArgs a,
                                                                      const __grid_constant__ TileMaps maps,
                                                                      const TileGeo geo) {
  static_assert(T == 16 || T == 32, "tokens per tile");
  constexpr int PLANE = T * 128;      // one [T tokens x 64 elements] bf16 plane
  constexpr int SB = TP_C * PLANE;    // bytes per ring slot (one box)
  constexpr int NST = TP_RING / SB;   // ring slots
  static_assert(NST % TP_NPH == 0 && NST <= TP_MAXST, "each slot serves one box phase");
  extern __shared__ uint8_t tp_smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(tp_smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* ring = smem;                                                              // [NST][SB]
  float* xbuf = reinterpret_cast<float*>(smem + TP_RING);                            // [NX][S][T][PS]
  float* red = xbuf + TP_NX * S * T * TP_PS;                                         // [phases][32][PS]
  float* alpha_s = red + TP_NPH * 32 * TP_PS;                                        // [NAB][T][4]
  __nv_bfloat16* wsl = reinterpret_cast<__nv_bfloat16*>(alpha_s + TP_NAB * T * 4);   // [M][wrow]
  __shared__ __align__(8) uint64_t full_bar[TP_MAXST];
  __shared__ __align__(8) uint64_t empty_bar[TP_MAXST];
  __shared__ __align__(8) uint64_t xfull[TP_NX];
  __shared__ __align__(8) uint64_t xdone[TP_NX];
  __shared__ __align__(8) uint64_t alpha_ready[TP_NAB];
  __shared__ __align__(8) uint64_t alpha_free[TP_NAB];
  __shared__ __align__(8) uint64_t wf_bar;
  __shared__ float bias_s[4];
  __shared__ volatile int abort_flag;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  pdl_launch_dependents();
  const uint32_t rank = cluster_rank(), cid = cluster_id_x(), ncl = n_clusters_x();
  const long long N = a.n_tokens;
  const int d = a.d, ec = geo.ec, ngrp = geo.ngrp, NB = M * ngrp;  // boxes per tile
  const long long nl = geo.ntiles > (long long)cid ? (geo.ntiles - cid + ncl - 1) / ncl : 0;

  if (tid < M) bias_s[tid] = a.b[tid];
  if (tid == 0) {
    // W_f slice, wsl[j][p*ec + e] = W_f[j][p*d + rank*ec + e]: one bulk copy
    // per (gate, path) run of ec elements, in flight beside the first boxes
    // of H (the gate warps wait for it once).  It is read before the wait on
    // the previous kernel: no kernel of this library writes W_f, and a kernel
    // from elsewhere (a caller's optimizer step) lets this one start only
    // when it completes, since it never triggers its dependents early.
    mbar_init(smem_u32(&wf_bar), 1);
    fence_mbar_init();
    mbar_arrive_expect_tx(smem_u32(&wf_bar), (uint32_t)(M * M * ec * 2));
    const __nv_bfloat16* Wf = reinterpret_cast<const __nv_bfloat16*>(a.Wf);
    for (int j = 0; j < M; ++j)
      for (int pth = 0; pth < M; ++pth)
        bulk_load(smem_u32(wsl + (size_t)j * geo.wrow + pth * ec),
                  Wf + (size_t)j * M * d + (size_t)pth * d + (size_t)rank * ec, (uint32_t)(ec * 2), smem_u32(&wf_bar));
    for (int i = 0; i < NST; ++i) {
      mbar_init(smem_u32(&full_bar[i]), 1);
      mbar_init(smem_u32(&empty_bar[i]), 2);  // the two gate warps of the box's phase
    }
    for (int i = 0; i < TP_NX; ++i) {
      mbar_init(smem_u32(&xfull[i]), 1);  // completes on the bytes of every sender
      mbar_init(smem_u32(&xdone[i]), 1);
    }
    for (int i = 0; i < TP_NAB; ++i) {
      mbar_init(smem_u32(&alpha_ready[i]), 1);
      mbar_init(smem_u32(&alpha_free[i]), TP_NWW);
    }
    abort_flag = 0;
    fence_mbar_init();
    for (int b = 0; b < TP_NX && b < nl; ++b) mbar_arrive_expect_tx(smem_u32(&xfull[b]), tp_xbytes(S, T));
  }
  __syncthreads();
  cluster_sync_all();  // every rank's barriers exist and are armed before anyone signals them
  pdl_wait();          // H and y may belong to the kernels before

  // a wait every lane of the warp takes; false for the whole warp on time-out
  // or when another role has given up
  auto warp_wait = [&](uint32_t bar, uint32_t parity, bool cluster_scope) -> bool {
    bool got = cluster_scope ? mbar_wait_cluster(bar, parity, a.status) : mbar_wait(bar, parity, a.status);
    got = __all_sync(0xffffffffu, got) && !__any_sync(0xffffffffu, abort_flag != 0);
    if (!got && lane == 0) abort_flag = 1;
    return got;
  };
  auto arrive = [&](uint64_t* bar) {
    if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
  };

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    long long g = 0;  // stages issued
    for (long long i = 0; i < nl; ++i) {
      const long long t0 = ((long long)cid + i * ncl) * T;
      bool ok = true;
      for (int j = 0; j < NB; ++j, ++g) {
        const int s = (int)(g % NST);
        if (!warp_wait(smem_u32(&empty_bar[s]), (uint32_t)((g / NST) & 1) ^ 1u, false)) {
          ok = false;
          break;
        }
        const int pth = j / ngrp, grp = j - pth * ngrp;
        if (lane == 0) {
          const bool last = grp == ngrp - 1;
          const uint32_t fb = smem_u32(&full_bar[s]);
          mbar_arrive_expect_tx(fb, (last ? geo.tail : TP_C) * PLANE);
          tma_load_3d(smem_u32(ring + s * SB), last ? &maps.tail : &maps.main, 0, (int)t0,
                      (pth * d + (int)rank * ec) / 64 + grp * TP_C, fb);
        }
        __syncwarp();
      }
      if (!ok) break;
    }
    // no copy may still be landing when the CTA exits
    for (long long k = g > NST ? g - NST : 0; k < g; ++k)
      if (!mbar_wait(smem_u32(&full_bar[k % NST]), (uint32_t)((k / NST) & 1), a.status)) break;
  } else if (warp <= TP_NGW) {
    // --------------------------------------------------------------- gates
    // warp (sub, hb) reads the boxes j with j % 4 == hb: with 32-token tiles
    // the 16 tokens 16*sub .. 16*sub + 15 of every plane, with 16-token tiles
    // all tokens of the planes c with c % 2 == sub
    const int gw = warp - 1, sub = gw & 1, hb = gw >> 1;  // hb 0..3
    const int g8 = lane >> 2, q = lane & 3;
    const __nv_bfloat16* wrowp = wsl + (size_t)(g8 < M ? g8 : 0) * geo.wrow + 2 * q;
    const int row = (T == 32 ? sub * 16 : 0) + (lane & 15), hsel = lane >> 4;
    // a failed W_f wait joins the first tile's decision below, so every gate
    // warp still meets the others at the named barrier
    const bool wf_ok = warp_wait(smem_u32(&wf_bar), 0u, false);
    for (long long i = 0; i < nl; ++i) {
      float acc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};  // two chains: plane parity
      // sums of squares as the diagonals of A A^T on the tensor cores: the B
      // fragment of A^T for tokens 0-7 is this thread's A registers 0 and 2,
      // for tokens 8-15 its registers 1 and 3
      float dl[4] = {0.f, 0.f, 0.f, 0.f}, dh[4] = {0.f, 0.f, 0.f, 0.f};
      bool ok = wf_ok;
      for (int j = hb; j < NB && ok; j += TP_NPH) {
        const long long gs = i * NB + j;  // stage counter
        const int s = (int)(gs % NST);
        if (!warp_wait(smem_u32(&full_bar[s]), (uint32_t)((gs / NST) & 1), false)) {
          ok = false;
          break;
        }
        const int pth = j / ngrp, grp = j - pth * ngrp;
        const int nc = grp == ngrp - 1 ? geo.tail : TP_C;
        const uint32_t sbase = smem_u32(ring + s * SB);
        const __nv_bfloat16* wk = wrowp + (pth * geo.nkb + grp * TP_C) * 64;
#pragma unroll
        for (int c = 0; c < TP_C; ++c) {
          if (c < nc && (T == 32 || (c & 1) == sub)) {
            // a plane's fragments first (loads in flight together), then its arithmetic
            uint32_t af[4][4], bf[4][2];
#pragma unroll
            for (int kk = 0; kk < 4; ++kk) {
              const int chunk = kk * 2 + hsel;
              ldsm_x4(sbase + c * PLANE + row * 128 + ((chunk ^ (row & 7)) << 4), af[kk][0], af[kk][1],
                      af[kk][2], af[kk][3]);
              bf[kk][0] = g8 < M ? *reinterpret_cast<const uint32_t*>(wk + c * 64 + kk * 16) : 0u;
              bf[kk][1] = g8 < M ? *reinterpret_cast<const uint32_t*>(wk + c * 64 + kk * 16 + 8) : 0u;
            }
#pragma unroll
            for (int kk = 0; kk < 4; ++kk) {
              mma16816(acc[kk & 1], af[kk], bf[kk][0], bf[kk][1]);
              mma16816(dl, af[kk], af[kk][0], af[kk][2]);
              mma16816(dh, af[kk], af[kk][1], af[kk][3]);
            }
          }
        }
        __syncwarp();
        arrive(&empty_bar[s]);
      }
      // this warp's [16 tokens][m + 1] partials into rows 16*sub.. of red[hb];
      // sender warps add the box phases (and with 16-token tiles the two plane
      // halves) in a fixed order and send one token row per lane to every rank
      float* rw = red + ((size_t)hb * 32 + sub * 16) * TP_PS;
      {
        // token g8's diagonal entry is column g8 of row g8: lane (g8, g8 / 2),
        // element 0 or 1 by parity; token g8 + 8's is row g8 + 8 of the
        // second product, elements 2 or 3
        const bool diag = (g8 >> 1) == q;
        const float s0 = (g8 & 1) ? dl[1] : dl[0];
        const float s1 = (g8 & 1) ? dh[3] : dh[2];
        if (2 * q < M) {
          rw[g8 * TP_PS + 2 * q] = acc[0][0] + acc[1][0];
          rw[(g8 + 8) * TP_PS + 2 * q] = acc[0][2] + acc[1][2];
        }
        if (2 * q + 1 < M) {
          rw[g8 * TP_PS + 2 * q + 1] = acc[0][1] + acc[1][1];
          rw[(g8 + 8) * TP_PS + 2 * q + 1] = acc[0][3] + acc[1][3];
        }
        if (diag) {
          rw[g8 * TP_PS + M] = s0;
          rw[(g8 + 8) * TP_PS + M] = s1;
        }
      }
      // one decision for the four gate warps (named barrier 3): all go on or all stop
      uint32_t go;
      asm volatile(
          "{\n .reg .pred p, q;\n setp.ne.u32 q, %1, 0;\n bar.red.and.pred p, 3, %2, q;\n selp.u32 %0, 1, 0, p;\n}\n"
          : "=r"(go)
          : "r"((uint32_t)ok), "n"(32 * TP_NGW)
          : "memory");
      if (!go) break;
      bool sent = true;
      if (hb == 0 && (T == 32 || sub == 0)) {
        // credit: this rank's alpha warp has read tile i - LA, so every rank
        // has read the buffer this tile's partials go to
        if (i >= TP_LA) {
          const long long c = i - TP_LA;
          sent = warp_wait(smem_u32(&xdone[c % TP_NX]), (uint32_t)((c / TP_NX) & 1), false);
        }
        if (sent && lane < 16) {
          const int b = (int)(i % TP_NX);
          const int tok = (T == 32 ? sub * 16 : 0) + lane;
          const float* r0 = red + (size_t)(T == 32 ? sub * 16 + lane : lane) * TP_PS;
          float4 lo = make_float4(0.f, 0.f, 0.f, 0.f), hi = lo;
#pragma unroll
          for (int h = 0; h < TP_NPH; ++h)  // the box phases in a fixed order
#pragma unroll
            for (int hs = 0; hs < (T == 32 ? 1 : 2); ++hs) {  // then the plane halves
              const float* rr = r0 + (h * 32 + hs * 16) * TP_PS;
              const float4 ah = *reinterpret_cast<const float4*>(rr);
              lo.x += ah.x;
              lo.y += ah.y;
              lo.z += ah.z;
              lo.w += ah.w;
              hi.x += rr[4];
            }
          const uint32_t lx = smem_u32(xbuf + (((size_t)b * S + rank) * T + tok) * TP_PS);
          const uint32_t lb = smem_u32(&xfull[b]);
#pragma unroll
          for (uint32_t r = 0; r < S; ++r) {
            st_async_v4(map_rank(lx, r), lo, map_rank(lb, r));
            st_async_v4(map_rank(lx + 16, r), hi, map_rank(lb, r));
          }
        }
        __syncwarp();
      }
      // red is rewritten only after every sender has read it
      asm volatile(
          "{\n .reg .pred p, q;\n setp.ne.u32 q, %1, 0;\n bar.red.and.pred p, 3, %2, q;\n selp.u32 %0, 1, 0, p;\n}\n"
          : "=r"(go)
          : "r"((uint32_t)sent), "n"(32 * TP_NGW)
          : "memory");
      if (!go) break;
    }
  } else if (warp == TP_NGW + 1) {
    // ---------------------------------------------------------------- alpha
    long long consumed = 0;
    bool ok = true;
    for (long long i = 0; i < nl; ++i) {
      consumed = i;
      const int b = (int)(i % TP_NX);
      if (!warp_wait(smem_u32(&xfull[b]), (uint32_t)((i / TP_NX) & 1), true)) {
        ok = false;
        break;
      }
      // lane = token: its partials from the ranks, summed in rank order
      float v[5] = {0.f, 0.f, 0.f, 0.f, 0.f};
      const int tl = lane < T ? lane : 0;  // lanes past the tile repeat token 0 and store nothing
#pragma unroll
      for (int r = 0; r < S; ++r) {
        const float* x = xbuf + (((size_t)b * S + r) * T + tl) * TP_PS;
        const float4 lo = *reinterpret_cast<const float4*>(x);
        v[0] += lo.x;
        v[1] += lo.y;
        v[2] += lo.z;
        v[3] += lo.w;
        v[4] += x[4];
      }
      __syncwarp();
      // buffer b is read: arm it for tile i + NX (no rank sends that tile
      // before this warp has read tile i + 2) and give the credit
      if (lane == 0 && i + TP_NX < nl) mbar_arrive_expect_tx(smem_u32(&xfull[b]), tp_xbytes(S, T));
      arrive(&xdone[b]);
      const int ab = (int)(i % TP_NAB);
      if (i >= TP_NAB && !warp_wait(smem_u32(&alpha_free[ab]), (uint32_t)(((i / TP_NAB) - 1) & 1), false)) {
        ok = false;
        break;
      }
      const float r = rsqrtf(v[M] / (float)(M * d) + a.rms_eps);
      float al[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int j = 0; j < M; ++j) al[j] = 1.0f / (1.0f + expf(-(a.gate_scale * r * v[j] + bias_s[j]))) + a.gate_offset;
      if (lane < T)
        *reinterpret_cast<float4*>(alpha_s + ((size_t)ab * T + lane) * 4) = make_float4(al[0], al[1], al[2], al[3]);
      const long long t = ((long long)cid + i * ncl) * T + lane;
      if (a.alpha_out && rank == 0 && lane < T && t < N)
#pragma unroll
        for (int j = 0; j < M; ++j) a.alpha_out[t * M + j] = al[j];
      __syncwarp();
      arrive(&alpha_ready[ab]);
    }
    if (!ok && lane == 0) {
      // abort: let the partials other ranks may still send land before the
      // cluster exits (one shared time limit for all of them)
      const unsigned long long tb = globaltimer_ns();
      for (long long j = consumed; j < nl && j < consumed + TP_NX; ++j) {
        const uint32_t bar = smem_u32(&xfull[j % TP_NX]), par = (uint32_t)((j / TP_NX) & 1);
        while (!mbar_try_wait_cluster(bar, par) && globaltimer_ns() - tb < kWaitLimitNs) {
        }
      }
    }
  } else {
    // ------------------------------------------------------- weighted warps
    const int ww = warp - TP_NGW - 2;
    const int vpt = ec / 8;            // 16-byte outputs per token in the slice
    const int nitems = T * vpt;
    const __nv_bfloat16* H = reinterpret_cast<const __nv_bfloat16*>(a.H);
    __nv_bfloat16* y = reinterpret_cast<__nv_bfloat16*>(a.y);
    for (long long i = 0; i < nl; ++i) {
      const int ab = (int)(i % TP_NAB);
      if (!warp_wait(smem_u32(&alpha_ready[ab]), (uint32_t)((i / TP_NAB) & 1), false)) break;
      const long long t0 = ((long long)cid + i * ncl) * T;
      const float* al_s = alpha_s + (size_t)ab * T * 4;
      for (int w0 = ww * 32 + lane; w0 < nitems; w0 += TP_NWW * 32 * TP_U) {
        uint4 h[TP_U][M];
        int tk[TP_U], col[TP_U];
#pragma unroll
        for (int r = 0; r < TP_U; ++r) {  // every load of the round before any arithmetic
          const int w = w0 + r * TP_NWW * 32;
          tk[r] = w / vpt;
          col[r] = (int)rank * ec + (w - tk[r] * vpt) * 8;
          const bool live = w < nitems && t0 + tk[r] < N;
          if (!live) tk[r] = -1;
#pragma unroll
          for (int p = 0; p < M; ++p)
            h[r][p] = live ? ld_stream16(H + ((t0 + tk[r]) * M + p) * d + col[r]) : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int r = 0; r < TP_U; ++r) {
          if (tk[r] < 0) continue;
          float out[8];
#pragma unroll
          for (int e = 0; e < 8; ++e) out[e] = 0.f;
#pragma unroll
          for (int p = 0; p < M; ++p) {
            float x[8];
            V16<__nv_bfloat16>::unpack(h[r][p], x);
            const float al = al_s[tk[r] * 4 + p];
#pragma unroll
            for (int e = 0; e < 8; ++e) out[e] = fmaf(al, x[e], out[e]);
          }
          *reinterpret_cast<uint4*>(y + (t0 + tk[r]) * d + col[r]) = V16<__nv_bfloat16>::pack(out);
        }
      }
      __syncwarp();  // alpha_s[ab] is free once every lane is past it
      arrive(&alpha_free[ab]);
    }
  }
  // the W_f copies have landed before the CTA exits, also when the gate
  // warps gave up first
  if (tid == 0) mbar_wait(smem_u32(&wf_bar), 0u, nullptr);
  __syncthreads();
  cluster_sync_all();  // no rank still writes into this CTA's shared memory
}

template <int M, int S, int T, int C>
cudaError_t launch_tile_mst(const ReduceArgs& a, const TileGeo& geo, size_t smem, const TileMaps* maps,
                            cudaStream_t s) {
  auto k = gated_reduce_tile_kernel<M, S, T, C>;
  cudaError_t e;
  int max_clusters = 0;
  if ((e = ensure_smem_limit((const void*)k, smem)) != cudaSuccess) return e;
  if ((e = max_active_clusters((const void*)k, TP_THR, smem, S, &max_clusters)) != cudaSuccess) return e;
  if (max_clusters < 1) return cudaErrorInvalidConfiguration;
  const long long ncl = std::min<long long>(max_clusters, geo.ntiles);
  return launch_kernel(k, dim3((unsigned)(ncl * S)), dim3(TP_THR), smem, s, (unsigned)S, a, *maps, geo);
}

// The tile geometries (CTAs per cluster, tokens per tile, chunks per box),
// in the order tile_geometry tries them, with the largest slice (bytes of
// H a CTA holds per tile) each may take.
struct TileShape {
  int s, t, c;
  int max_slice_kb;
};
constexpr TileShape kTileShapes[] = {{4, 32, 8, 160}, {4, 16, 8, 240}, {8, 16, 8, 240}, {4, 32, 4, 300},
                                     {8, 32, 4, 300}, {4, 16, 4, 300}, {8, 16, 4, 300}};

template <int M>
cudaError_t launch_tile_m(const ReduceArgs& a, const TileGeo& geo, size_t smem, const TileMaps* maps,
                          cudaStream_t s) {
  const int code = geo.s * 1000 + geo.t * 10 + geo.c;
  switch (code) {
    case 4328: return launch_tile_mst<M, 4, 32, 8>(a, geo, smem, maps, s);
    case 4168: return launch_tile_mst<M, 4, 16, 8>(a, geo, smem, maps, s);
    case 8168: return launch_tile_mst<M, 8, 16, 8>(a, geo, smem, maps, s);
    case 4324: return launch_tile_mst<M, 4, 32, 4>(a, geo, smem, maps, s);
    case 8324: return launch_tile_mst<M, 8, 32, 4>(a, geo, smem, maps, s);
    case 4164: return launch_tile_mst<M, 4, 16, 4>(a, geo, smem, maps, s);
    case 8164: return launch_tile_mst<M, 8, 16, 4>(a, geo, smem, maps, s);
    default: return cudaErrorInvalidValue;
  }
}

// The weighted pass re-reads a CTA's slice of a tile from L2, so the slice
// must stay in it (with 4-CTA clusters and 32 tokens at m = 4, d = 7168, 459
// KB slices, the launch read 800 MB from DRAM for 470 MB of H).  The
// geometry is the first of kTileShapes whose slice fits its limit, whose
// boxes per tile are a whole number of phases and whose shared memory fits.
// It depends on m and d only, never on the token count.  Measured on GB300
// (m = 4, TB/s): 4-CTA clusters keep 144 SMs busy where 8-CTA clusters of
// this CTA keep 120; boxes of 8 chunks (1 KB contiguous per token) beat 4:
//   d = 7168, 131072 tokens: (8, 32, 4) 4.10, (4, 16, 8) 4.87
//   d = 4096, 139264 tokens: (4, 32, 4) 3.92, (4, 16, 8) 5.18
//   d = 2048,   2048 tokens: (4, 32, 4) 2.46, (4, 32, 8) 2.71 (65536: 5.09, 4.64)
bool tile_geometry(const ReduceArgs& a, int dtype, TileGeo* geo, size_t* smem) {
  if (dtype != HDF_BF16 || a.alpha_override || a.path_norm_w) return false;
  if (a.n_tokens <= 0 || a.n_tokens > (1ll << 31) - 64) return false;  // TMA coordinates are 32-bit
  if (!(a.m == 1 || a.m == 2 || a.m == 4)) return false;
  for (const TileShape& sh : kTileShapes) {
    const int S = sh.s;
    if (a.d % (S * 64)) continue;
    geo->s = S;
    geo->ec = a.d / S;
    geo->t = sh.t;
    geo->c = sh.c;
    if ((size_t)geo->t * a.m * geo->ec * 2 > (size_t)sh.max_slice_kb * 1024) continue;
    geo->nkb = geo->ec / 64;
    geo->ngrp = (geo->nkb + geo->c - 1) / geo->c;
    geo->tail = geo->nkb - (geo->ngrp - 1) * geo->c;
    if ((a.m * geo->ngrp) % TP_NPH) continue;  // boxes per tile: a multiple of the 4 phases
    geo->wrow = a.m * geo->ec + 8;  // + 16 bytes: the gate rows of one B fragment sit in distinct banks
    geo->ntiles = (a.n_tokens + geo->t - 1) / geo->t;
    *smem = tp_smem(S, geo->t, a.m, geo->wrow);
    if (*smem <= 227 * 1024) return true;
  }
  return false;
}

}  // namespace

bool reduce_tile_boxes(const ReduceArgs& a, int dtype, unsigned box[3], unsigned tail_box[3]) {
  TileGeo geo;
  size_t smem;
  if (!tile_geometry(a, dtype, &geo, &smem)) return false;
  box[0] = tail_box[0] = 64;
  box[1] = tail_box[1] = (unsigned)geo.t;
  box[2] = (unsigned)std::min(geo.c, geo.nkb);
  tail_box[2] = (unsigned)geo.tail;
  return true;
}

cudaError_t launch_gated_reduce_tile(const ReduceArgs& a, const CUtensorMap* maps2, cudaStream_t s) {
  TileGeo geo;
  size_t smem;
  if (!tile_geometry(a, HDF_BF16, &geo, &smem)) return cudaErrorInvalidValue;
  TileMaps maps;
  maps.main = maps2[0];
  maps.tail = maps2[1];
  switch (a.m) {
    case 1: return launch_tile_m<1>(a, geo, smem, &maps, s);
    case 2: return launch_tile_m<2>(a, geo, smem, &maps, s);
    case 4: return launch_tile_m<4>(a, geo, smem, &maps, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace hdf
