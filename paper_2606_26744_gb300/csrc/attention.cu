// Non-causal block attention of the drafter (anchor-plus-mask block over the
// reduced target context; Sec. 2.1 of the HyperDFlash paper as read for the
// DFlash-style drafter): for sequence b and head h,
//   O = softmax(Q [K_c; K_b]^T / sqrt(hd)) [V_c; V_b]
// with the B block queries attending to all T_b context keys and all B block
// keys, nothing across sequences.
//
// bf16 path (split-KV, flash-decoding style): grid (chunk, head, sequence).
// A producer warp streams 64-key K/V tiles with TMA (128-byte swizzle) into a
// 4-stage ring; tile i lands in stage i % 4 and is consumed by warp i % 4,
// which runs S = Q K^T and O += P V on mma.sync m16n8k16 (the B <= 16 queries
// are one m16 row tile) with an fp32 online softmax in the log2 domain.  The
// four warps merge in shared memory.  With one chunk per (sequence, head)
// that is the output; with several (at most 8) the chunks of one (sequence,
// head) are one thread-block cluster: each CTA leaves its fp32 partial
// (m, l, O) in its shared memory and, after a cluster barrier, each merges a
// slice of the block rows over all chunks in chunk order, over DSMEM.
// With B queries per key the kernel does ~B flops per byte of K/V, so it is
// bound by HBM, not by the tensor pipe.
#include <atomic>
#include <cmath>

#include "common.cuh"
#include "kernels.h"

namespace hdf {
namespace {

constexpr int KT = 64;       // keys per tile
constexpr int NSTAGE = 4;
constexpr int NCW = 4;       // consumer warps
// Tile t goes to stage t % NSTAGE and to consumer warp t % NCW: with the two
// equal, each warp waits only on its own stage, one fill at a time.  A warp
// that could wait on a stage two fills ahead would pass the parity wait on
// the older fill (mbarrier parity tells adjacent phases apart only).
static_assert(NSTAGE == NCW, "stage / consumer-warp affinity");

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                          uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
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

// First row and key count of sequence b's context: packed rows from cu_ctx,
// or the cached rows b * ctx_stride + [0, ctx_len[b]).  A cached length
// outside [0, max_len] is limited to it and recorded (by one thread).
__device__ __forceinline__ void context_span(const AttnArgs& a, int b, bool report, int* c0, int* T) {
  if (a.ctx_len) {
    int t = a.ctx_len[b];
    if (t < 0 || t > a.max_len) {
      if (report) record_device_error(a.status);
      t = t < 0 ? 0 : a.max_len;
    }
    *c0 = (int)(b * a.ctx_stride);
    *T = t;
  } else {
    *c0 = a.cu_ctx[b];
    *T = a.cu_ctx[b + 1] - *c0;
  }
}

// byte offset of the 16-byte chunk c (0..7) of row r in a 128-byte-swizzled box
__device__ __forceinline__ uint32_t sw128(int r, int c) {
  return (uint32_t)(r * 128 + ((c ^ (r & 7)) << 4));
}

template <int HD>
__global__ void __launch_bounds__(160, 1)
    attn_bf16_kernel(const AttnArgs a, const __grid_constant__ AttnTmaps tm) {
  constexpr int HALVES = HD / 64;
  constexpr int TILE_BYTES = HALVES * KT * 128;   // one of K or V
  constexpr int STAGE_BYTES = 2 * TILE_BYTES;
  constexpr int NB_O = HD / 8;                     // n-blocks of the output
  constexpr int KS = HD / 16;                      // k-steps of Q K^T
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  __shared__ __align__(8) uint64_t full_bar[NSTAGE];
  __shared__ __align__(8) uint64_t empty_bar[NSTAGE];
  __shared__ float wm[NCW][16], wl[NCW][16];

  const int chunk_id = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  pdl_launch_dependents();
  const int B = a.block;
  if (tid == 0) {
    for (int s = 0; s < NSTAGE; ++s) {
      mbar_init(smem_u32(&full_bar[s]), 1);
      mbar_init(smem_u32(&empty_bar[s]), 1);
    }
    fence_mbar_init();
  }
  __syncthreads();
  pdl_wait();  // Q, the block / context K, V and the cache lengths come from the kernels before
  int c0, T;
  context_span(a, b, chunk_id == 0 && h == 0 && tid == 0, &c0, &T);
  // chunks past the sequence's keys hold no tiles: in a cluster they still
  // join its barriers, with an empty partial (m = -inf, l = 0)
  const int nc_b = min(a.n_chunks, T > 0 ? (T + a.chunk - 1) / a.chunk : 1);
  const int kbeg = chunk_id * a.chunk;
  const int kend = min(T, kbeg + a.chunk);
  const int n_ctx_tiles = kend > kbeg ? (kend - kbeg + KT - 1) / KT : 0;
  const bool has_block = chunk_id == nc_b - 1;
  const int ntiles = n_ctx_tiles + (has_block ? 1 : 0);

  if (warp == NCW) {
    if (lane == 0) {  // ------------------------------------------ producer
      for (int t = 0; t < ntiles; ++t) {
        const int s = t % NSTAGE;
        const uint32_t ph = (t / NSTAGE) & 1;
        if (!mbar_wait(smem_u32(&empty_bar[s]), ph ^ 1, a.status)) break;
        const uint32_t fb = smem_u32(&full_bar[s]);
        mbar_arrive_expect_tx(fb, STAGE_BYTES);
        const uint32_t base = smem_u32(smem + s * STAGE_BYTES);
        const bool blk = t >= n_ctx_tiles;
        const CUtensorMap* mk = blk ? &tm.kb : &tm.k;
        const CUtensorMap* mv = blk ? &tm.vb : &tm.v;
        const int row0 = blk ? b * B : c0 + kbeg + t * KT;
#pragma unroll
        for (int hh = 0; hh < HALVES; ++hh) {
          tma_load_2d(base + hh * KT * 128, mk, h * HD + hh * 64, row0, fb);
          tma_load_2d(base + TILE_BYTES + hh * KT * 128, mv, h * HD + hh * 64, row0, fb);
        }
      }
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ consumers
    const int g = lane >> 2, q = lane & 3;
    const float scale = rsqrtf((float)HD) * 1.4426950408889634f;  // log2(e)/sqrt(hd)
    uint32_t qa[KS][4];
    {
      const __nv_bfloat16* Q = reinterpret_cast<const __nv_bfloat16*>(a.q);
      const long long r0 = (long long)b * B + g, r1 = r0 + 8;
      const bool v0 = g < B, v1 = g + 8 < B;
#pragma unroll
      for (int ks = 0; ks < KS; ++ks) {
        const int col = h * HD + ks * 16 + 2 * q;
        qa[ks][0] = v0 ? *reinterpret_cast<const uint32_t*>(Q + r0 * a.d + col) : 0u;
        qa[ks][1] = v1 ? *reinterpret_cast<const uint32_t*>(Q + r1 * a.d + col) : 0u;
        qa[ks][2] = v0 ? *reinterpret_cast<const uint32_t*>(Q + r0 * a.d + col + 8) : 0u;
        qa[ks][3] = v1 ? *reinterpret_cast<const uint32_t*>(Q + r1 * a.d + col + 8) : 0u;
      }
    }
    float o[NB_O][4];
#pragma unroll
    for (int i = 0; i < NB_O; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
    float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;

    for (int t = warp; t < ntiles; t += NCW) {
      const int s = t % NSTAGE;
      const uint32_t ph = (t / NSTAGE) & 1;
      const bool got = mbar_wait(smem_u32(&full_bar[s]), ph, a.status);
      if (!__all_sync(0xffffffffu, got)) break;  // warp-uniform exit
      const bool blk = t >= n_ctx_tiles;
      const int valid = blk ? B : min(KT, kend - kbeg - t * KT);
      const uint32_t kbase = smem_u32(smem + s * STAGE_BYTES);
      const uint32_t vbase = kbase + TILE_BYTES;
      if (a.ctx_len && !blk && valid < KT) {
        // cache rows past the sequence's length may hold anything; their
        // softmax weight is 0, so zero their V for an exact 0 contribution
        uint8_t* vt = smem + s * STAGE_BYTES + TILE_BYTES;
        for (int i = lane; i < (KT - valid) * HALVES * 8; i += 32) {
          const int r = valid + i / (HALVES * 8), rem = i % (HALVES * 8);
          *reinterpret_cast<uint4*>(vt + (rem >> 3) * (KT * 128) + r * 128 + (rem & 7) * 16) = make_uint4(0, 0, 0, 0);
        }
        // the stage is refilled by TMA (async proxy) after these generic stores
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        __syncwarp();
      }

      // S = Q K^T for 64 keys: 8 n-blocks of 8 keys
      float sc[8][4];
#pragma unroll
      for (int nb = 0; nb < 8; ++nb) {
        sc[nb][0] = sc[nb][1] = sc[nb][2] = sc[nb][3] = 0.f;
#pragma unroll
        for (int kp = 0; kp < KS / 2; ++kp) {
          const int mat = lane >> 3, rr = lane & 7;
          const int key = nb * 8 + rr;
          const int cg = 4 * kp + mat;  // 16-byte chunk along hd
          const uint32_t addr = kbase + (cg >> 3) * (KT * 128) + sw128(key, cg & 7);
          uint32_t b0, b1, b2, b3;
          ldsm_x4(addr, b0, b1, b2, b3);
          mma16816(sc[nb], qa[2 * kp], b0, b1);
          mma16816(sc[nb], qa[2 * kp + 1], b2, b3);
        }
      }
      // mask and scale, row maxima (rows g and g+8)
      float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
      for (int nb = 0; nb < 8; ++nb) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int key = nb * 8 + 2 * q + (e & 1);
          const float v = key < valid ? sc[nb][e] * scale : -INFINITY;
          sc[nb][e] = v;
        }
        mx0 = fmaxf(mx0, fmaxf(sc[nb][0], sc[nb][1]));
        mx1 = fmaxf(mx1, fmaxf(sc[nb][2], sc[nb][3]));
      }
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
      const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
      const float al0 = exp2f(m0 - mn0), al1 = exp2f(m1 - mn1);
      m0 = mn0;
      m1 = mn1;
      float ps0 = 0.f, ps1 = 0.f;
#pragma unroll
      for (int nb = 0; nb < 8; ++nb) {
        sc[nb][0] = exp2f(sc[nb][0] - mn0);
        sc[nb][1] = exp2f(sc[nb][1] - mn0);
        sc[nb][2] = exp2f(sc[nb][2] - mn1);
        sc[nb][3] = exp2f(sc[nb][3] - mn1);
        ps0 += sc[nb][0] + sc[nb][1];
        ps1 += sc[nb][2] + sc[nb][3];
      }
      l0 = l0 * al0 + ps0;
      l1 = l1 * al1 + ps1;
#pragma unroll
      for (int i = 0; i < NB_O; ++i) {
        o[i][0] *= al0; o[i][1] *= al0;
        o[i][2] *= al1; o[i][3] *= al1;
      }
      // O += P V : 4 k-steps of 16 keys.  P is split into a bf16 high part
      // and a bf16 remainder (two MMAs), which keeps ~16 significant bits of
      // the softmax weights instead of bf16's 8.
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        uint32_t pa[4], pl[4];
        const float pv8[8] = {sc[2 * kk][0], sc[2 * kk][1], sc[2 * kk][2], sc[2 * kk][3],
                              sc[2 * kk + 1][0], sc[2 * kk + 1][1], sc[2 * kk + 1][2], sc[2 * kk + 1][3]};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          pa[i] = pack_bf16x2(pv8[2 * i], pv8[2 * i + 1]);
          pl[i] = pack_bf16x2(pv8[2 * i] - bf16lo(pa[i]), pv8[2 * i + 1] - bf16hi(pa[i]));
        }
#pragma unroll
        for (int np = 0; np < NB_O / 2; ++np) {
          const int mat = lane >> 3, rr = lane & 7;
          const int key = kk * 16 + (mat & 1) * 8 + rr;
          const int cg = 2 * np + (mat >> 1);
          const uint32_t addr = vbase + (cg >> 3) * (KT * 128) + sw128(key, cg & 7);
          uint32_t b0, b1, b2, b3;
          ldsm_x4_t(addr, b0, b1, b2, b3);
          mma16816(o[2 * np], pa, b0, b1);
          mma16816(o[2 * np], pl, b0, b1);
          mma16816(o[2 * np + 1], pa, b2, b3);
          mma16816(o[2 * np + 1], pl, b2, b3);
        }
      }
      __syncwarp();
      if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(&empty_bar[s])) : "memory");
    }
    l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
    l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
    if (q == 0) {
      wm[warp][g] = m0; wl[warp][g] = l0;
      wm[warp][g + 8] = m1; wl[warp][g + 8] = l1;
    }
    __syncthreads();  // (A) every consumer is done with the stage ring
    float* ow = reinterpret_cast<float*>(smem);  // [NCW][16][HD]
#pragma unroll
    for (int i = 0; i < NB_O; ++i) {
      const int col = i * 8 + 2 * q;
      ow[(warp * 16 + g) * HD + col] = o[i][0];
      ow[(warp * 16 + g) * HD + col + 1] = o[i][1];
      ow[(warp * 16 + g + 8) * HD + col] = o[i][2];
      ow[(warp * 16 + g + 8) * HD + col + 1] = o[i][3];
    }
  }
  if (warp == NCW) __syncthreads();  // matches (A)
  __syncthreads();

  // merge the four warps into this chunk's (m, l, O): one factor per (warp,
  // row), then the element sums over the warps in order, 4 columns per thread
  __shared__ float fw[NCW][16], pm[16], pl[16];
  if (tid < B) {
    float mstar = -INFINITY;
#pragma unroll
    for (int w = 0; w < NCW; ++w) mstar = fmaxf(mstar, wm[w][tid]);
    float lsum = 0.f;
#pragma unroll
    for (int w = 0; w < NCW; ++w) {
      const float f = wm[w][tid] == -INFINITY ? 0.f : exp2f(wm[w][tid] - mstar);
      fw[w][tid] = f;
      lsum += wl[w][tid] * f;
    }
    pm[tid] = mstar;
    pl[tid] = lsum;
  }
  __syncthreads();
  const float* ow = reinterpret_cast<const float*>(smem);
  __nv_bfloat16* out = reinterpret_cast<__nv_bfloat16*>(a.out);
  const int nc = (int)gridDim.x;  // chunks per (sequence, head): the cluster size
  float* po = reinterpret_cast<float*>(smem + NCW * 16 * HD * 4);  // [16][HD] partial O, unnormalised
  constexpr int C4 = HD / 4;
  for (int i = tid; i < B * C4; i += blockDim.x) {
    const int r = i / C4, c4 = i - r * C4;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int w = 0; w < NCW; ++w) {
      const float4 x = *reinterpret_cast<const float4*>(ow + (w * 16 + r) * HD + 4 * c4);
      const float f = fw[w][r];
      acc.x += x.x * f;
      acc.y += x.y * f;
      acc.z += x.z * f;
      acc.w += x.w * f;
    }
    if (nc == 1) {
      const float l = pl[r];
      uint2 pk;
      pk.x = pack_bf16x2(acc.x / l, acc.y / l);
      pk.y = pack_bf16x2(acc.z / l, acc.w / l);
      *reinterpret_cast<uint2*>(out + ((size_t)b * B + r) * a.d + h * HD + 4 * c4) = pk;
    } else {
      *reinterpret_cast<float4*>(po + r * HD + 4 * c4) = acc;
    }
  }
  if (nc == 1) return;

  // O = sum_c O_c 2^(m_c - m*) / sum_c l_c 2^(m_c - m*) over the chunks c of
  // the cluster, in chunk order; rank r merges block rows [r * rpr, (r+1) * rpr)
  cluster_sync_all();  // every chunk's partial is in its shared memory
  {
    const int rank = (int)cluster_rank();
    const int rpr = (B + nc - 1) / nc;
    const int r0 = rank * rpr, nr = max(0, min(B, r0 + rpr) - r0);
    for (int it = tid; it < nr * C4; it += blockDim.x) {
      const int r = r0 + it / C4, c4 = it - (it / C4) * C4;
      float mc[8], lc[8];
#pragma unroll
      for (int c = 0; c < 8; ++c)
        if (c < nc) {
          mc[c] = ld_dsmem_f32(map_rank(smem_u32(&pm[r]), (uint32_t)c));
          lc[c] = ld_dsmem_f32(map_rank(smem_u32(&pl[r]), (uint32_t)c));
        }
      float mstar = -INFINITY;
#pragma unroll
      for (int c = 0; c < 8; ++c)
        if (c < nc) mstar = fmaxf(mstar, mc[c]);
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
      float l = 0.f;
#pragma unroll
      for (int c = 0; c < 8; ++c)
        if (c < nc && mc[c] != -INFINITY) {  // -inf: a chunk without keys of this sequence
          const float f = exp2f(mc[c] - mstar);
          const float4 q = ld_dsmem_v4(map_rank(smem_u32(po + r * HD + 4 * c4), (uint32_t)c));
          acc.x += q.x * f;
          acc.y += q.y * f;
          acc.z += q.z * f;
          acc.w += q.w * f;
          l += lc[c] * f;
        }
      uint2 pk;
      pk.x = pack_bf16x2(acc.x / l, acc.y / l);
      pk.y = pack_bf16x2(acc.z / l, acc.w / l);
      *reinterpret_cast<uint2*>(out + ((size_t)b * B + r) * a.d + h * HD + 4 * c4) = pk;
    }
  }
  cluster_sync_all();  // no CTA leaves while another still reads its shared memory
}

// fp32 path (tiny correctness workloads): one warp per (sequence, head, query),
// exact online softmax over the keys, lane-parallel along head_dim.
__global__ void attn_f32_kernel(const AttnArgs a) {
  pdl_launch_dependents();
  pdl_wait();
  const int h = blockIdx.x, b = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int HD = a.head_dim;
  const float* Q = reinterpret_cast<const float*>(a.q);
  const float* Kc = reinterpret_cast<const float*>(a.kc);
  const float* Vc = reinterpret_cast<const float*>(a.vc);
  const float* Kb = reinterpret_cast<const float*>(a.kb);
  const float* Vb = reinterpret_cast<const float*>(a.vb);
  float* out = reinterpret_cast<float*>(a.out);
  int c0, T;
  context_span(a, b, h == 0 && threadIdx.x == 0, &c0, &T);
  const float scale = rsqrtf((float)HD);
  for (int r = warp; r < a.block; r += blockDim.x >> 5) {
    const size_t qrow = (size_t)b * a.block + r;
    float qv[4], acc[4] = {0.f, 0.f, 0.f, 0.f};
    for (int e = 0; e < 4; ++e) {
      const int c = lane + 32 * e;
      qv[e] = c < HD ? Q[qrow * a.d + h * HD + c] : 0.f;
    }
    float m = -INFINITY, l = 0.f;
    for (int j = 0; j < T + a.block; ++j) {
      const float* kr = j < T ? Kc + (size_t)(c0 + j) * a.d : Kb + ((size_t)b * a.block + j - T) * a.d;
      const float* vr = j < T ? Vc + (size_t)(c0 + j) * a.d : Vb + ((size_t)b * a.block + j - T) * a.d;
      float s = 0.f;
      for (int e = 0; e < 4; ++e) {
        const int c = lane + 32 * e;
        if (c < HD) s += qv[e] * kr[h * HD + c];
      }
      s = warp_sum(s) * scale;
      const float mn = fmaxf(m, s);
      const float al = expf(m - mn), p = expf(s - mn);
      l = l * al + p;
      for (int e = 0; e < 4; ++e) {
        const int c = lane + 32 * e;
        acc[e] = acc[e] * al + (c < HD ? p * vr[h * HD + c] : 0.f);
      }
      m = mn;
    }
    for (int e = 0; e < 4; ++e) {
      const int c = lane + 32 * e;
      if (c < HD) out[qrow * a.d + h * HD + c] = acc[e] / l;
    }
  }
}

template <int HD>
constexpr size_t attn_smem() { return (size_t)NSTAGE * 2 * (HD / 64) * KT * 128 + 1024; }

template <int HD>
cudaError_t launch_hd(const AttnArgs& a, const AttnTmaps* tm, cudaStream_t s) {
  auto k = attn_bf16_kernel<HD>;
  cudaError_t e;
  if ((e = ensure_smem_limit((const void*)k, attn_smem<HD>())) != cudaSuccess) return e;
  if (a.n_chunks < 1 || a.n_chunks > 8) return cudaErrorInvalidValue;
  // the chunks of one (sequence, head) are one cluster
  return launch_kernel(k, dim3(a.n_chunks, a.n_heads, a.batch), dim3(160), attn_smem<HD>(), s,
                       (unsigned)a.n_chunks, a, *tm);
}

}  // namespace

size_t attention_smem_bytes(int head_dim) { return head_dim == 64 ? attn_smem<64>() : attn_smem<128>(); }

// Clusters of `cluster` attention CTAs resident at once on the current device
// (occupancy API), or -1 if it cannot be asked (or answers none).
int attention_max_clusters(int head_dim, int cluster) {
  if ((head_dim != 64 && head_dim != 128) || cluster < 1 || cluster > 8) return -1;
  const bool hi = head_dim == 128;
  const void* k = hi ? (const void*)attn_bf16_kernel<128> : (const void*)attn_bf16_kernel<64>;
  const size_t smem = hi ? attn_smem<128>() : attn_smem<64>();
  int n = 0;
  if (ensure_smem_limit(k, smem) != cudaSuccess || max_active_clusters(k, 160, smem, cluster, &n) != cudaSuccess) {
    cudaGetLastError();
    return -1;
  }
  return n > 0 ? n : -1;  // none: the caller falls back to SMs / cluster size
}

cudaError_t launch_attention(const AttnArgs& a, const AttnTmaps* tm, int dtype, cudaStream_t s) {
  if (a.batch == 0) return cudaSuccess;
  if (dtype == HDF_F32) {
    return launch_kernel(attn_f32_kernel, dim3(a.n_heads, a.batch), dim3(128), 0, s, 1u, a);
  }
  if (a.head_dim == 64) return launch_hd<64>(a, tm, s);
  if (a.head_dim == 128) return launch_hd<128>(a, tm, s);
  return cudaErrorInvalidValue;
}

}  // namespace hdf
