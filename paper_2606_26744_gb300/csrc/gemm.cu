// tcgen05 / TMEM GEMM for the dense contractions of the draft step:
// the conditioning projection (context K/V), the block Q/K/V/O projections,
// the SwiGLU MLP and the LM head (Sec. 2.1-2.3 of the HyperDFlash paper as
// read for the drafter), plus the generic fc reducer of Table 1.
//
//   D[M, N] = A[M, K] * B[N, K]^T      (both operands K-major)
//
// One CTA of 4 warps computes a 128 x BN tile (optionally one K-split of it):
//   warp 0 / lane 0  TMA producer: A as two 64-row boxes, B as one BN-row box,
//                    128-byte swizzle, into a STAGES-deep shared-memory ring
//   warp 1 / lane 0  MMA issuer: tcgen05.mma.cta_group::1 (kind::f16 for bf16,
//                    kind::tf32 for fp32), 4 MMAs of K=16 (bf16) per stage,
//                    fp32 accumulator in TMEM, tcgen05.commit frees the stage
//   warp 2           TMEM allocation / release
//   all 4 warps      epilogue: tcgen05.ld 32x32b (thread i <-> TMEM lane i =
//                    tile row i), fused RoPE / residual add / SwiGLU / LM-head
//                    argmax + sum-exp partials, direct global stores.
// Split-K: the k_splits CTAs of a tile form one thread-block cluster.  Each
// leaves its fp32 partial tile in its own shared memory; after a cluster
// barrier every rank sums one slice of the tile's rows over all ranks, in
// rank order, over distributed shared memory, and writes the sums into rank
// 0's partial tile in place (no other rank reads that slice); after a second
// barrier rank 0 runs the epilogue.  No global round trip, no atomics.
#include <algorithm>
#include <atomic>
#include <climits>

#include "common.cuh"
#include "kernels.h"

namespace hdf {
namespace {

constexpr int BM = 128;
constexpr int ROW_BYTES = 128;  // one 128-byte swizzle row per tile row and stage

template <typename T> struct GT;
template <> struct GT<__nv_bfloat16> {
  static constexpr int BK = 64;
  static constexpr uint32_t FMT = 1;  // bf16
};
template <> struct GT<float> {
  static constexpr int BK = 32;
  static constexpr uint32_t FMT = 2;  // tf32
};

// Rings of ~96 KB, so that two CTAs share an SM: two independent producers
// keep more loads in flight than one CTA with a ring twice as deep
// (measured on the skinny weight-streaming GEMMs of the draft step).
constexpr int stages_for(int bn) { return bn >= 224 ? 2 : (bn >= 128 ? 3 : (bn >= 64 ? 4 : 5)); }
constexpr int kPartialOffset = 12288;  // split-K partial tile (rank 0's is reduced in place), in the drained
                                       // stage memory above the epilogue's scratch (at most 16 x 136 floats)
constexpr bool partial_fits(int bn) { return kPartialOffset + BM * bn * 4 <= stages_for(bn) * (BM + bn) * ROW_BYTES; }
static_assert(partial_fits(16) && partial_fits(32) && partial_fits(64) && partial_fits(128),
              "split-K partial tile fits the stage memory (BN <= 128)");
constexpr int smem_for(int bn) { return stages_for(bn) * (BM + bn) * ROW_BYTES + 1024; }

__device__ __forceinline__ void operand_rows(const Operand& op, int tile_row0, int half, int tile_idx,
                                             const CUtensorMap** map, int* row) {
  if (op.mode == kPair64) {
    *map = &op.map[half];
    *row = tile_idx * 64;
  } else {
    const int r = tile_row0 + half * 64;
    const int mi = r / op.rows_per_map;
    *map = &op.map[mi];
    *row = r - mi * op.rows_per_map;
  }
}

__device__ __forceinline__ int ctx_position(const int* cu, int batch, long long t) {
  int lo = 0, hi = batch;  // find b with cu[b] <= t < cu[b+1]
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (__ldg(cu + mid) <= t) lo = mid; else hi = mid;
  }
  return (int)(t - __ldg(cu + lo));
}
__device__ __forceinline__ int block_position(const Epilogue& E, int j) {
  const int b = j / E.block;
  const int n = E.pos_mode == 4 ? 0 : __ldg(E.cu_ctx + b + 1) - __ldg(E.cu_ctx + b);
  const int T = E.pos_mode >= 4 ? __ldg(E.ctx_len + b) + n : n;
  return T + (j - b * E.block);
}

// Context row t of a kEpiStore GEMM: its output row (or -1: not stored) and
// its RoPE position.  Mode 3 appends to a cache: sequence b's rows go after
// the ctx_len[b] rows it already holds, rows past cu[batch] are skipped, and
// a row that would pass the cache capacity is skipped and recorded.
__device__ __forceinline__ long long ctx_store_row(const Epilogue& E, long long t, int* pos, int* status) {
  if (E.pos_mode == 1) {
    *pos = ctx_position(E.cu_ctx, E.batch, t);
    return t;
  }
  if (E.pos_mode != 3) {
    *pos = 0;
    return t;
  }
  *pos = 0;
  if (t >= __ldg(E.cu_ctx + E.batch)) return -1;
  int lo = 0, hi = E.batch;
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (__ldg(E.cu_ctx + mid) <= t) lo = mid; else hi = mid;
  }
  const long long p = (long long)__ldg(E.ctx_len + lo) + (t - __ldg(E.cu_ctx + lo));
  if (p < 0 || p >= E.cache_cap) {
    record_device_error(status);
    return -1;
  }
  *pos = (int)p;
  return (long long)lo * E.cache_cap + p;
}

// Token column j of a kEpiStoreT GEMM: its output row (or -1: not stored)
// and its RoPE position.  Context rows (modes 1 and 3) as ctx_store_row;
// block rows land at row j, at their block position.
__device__ __forceinline__ long long column_target(const Epilogue& E, long long j, int* pos, int* status) {
  if (E.pos_mode == 1 || E.pos_mode == 3) return ctx_store_row(E, j, pos, status);
  *pos = E.pos_mode == 0 ? 0 : block_position(E, (int)j);
  return j;
}

template <typename T>
__device__ __forceinline__ void store16(T* dst, const float* v);
template <>
__device__ __forceinline__ void store16<__nv_bfloat16>(__nv_bfloat16* dst, const float* v) {
  uint4* p = reinterpret_cast<uint4*>(dst);
  p[0] = V16<__nv_bfloat16>::pack(v);
  p[1] = V16<__nv_bfloat16>::pack(v + 8);
}
template <>
__device__ __forceinline__ void store16<float>(float* dst, const float* v) {
  float4* p = reinterpret_cast<float4*>(dst);
#pragma unroll
  for (int i = 0; i < 4; ++i) p[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
}

// Epilogue for one 16-column chunk of the tile.  Called by all 128 threads
// with identical (tile, c0) so that shuffles and barriers are uniform.
// rope_row: this thread's row of the RoPE table staged in shared memory
// (cos of the hd/2 pairs, then sin, see stage_rope_row), or nullptr.
// srow: kEpiStore output row of this thread's token from ctx_store_row (-1:
// not stored).
template <typename T, int BN>
__device__ __forceinline__ void epilogue_chunk(const GemmArgs& g, int tile_m, int tile_n, int c0,
                                               float* v, uint8_t* smem, const float* rope_row, long long srow,
                                               int spos) {
  const Epilogue& E = g.epi;
  const int row = threadIdx.x;
  const int lane = row & 31, warp = row >> 5;
  switch (E.kind) {
    case kEpiStore: {  // rows = tokens, columns = output features
      const long long t = (long long)tile_m * BM + row;
      const int col0 = tile_n * BN + c0;
      if (t >= g.M || col0 >= g.N || srow < 0) return;
      const int seg = col0 / E.seg_width;
      const int fl = col0 - seg * E.seg_width;
      if ((E.rope_mask >> seg) & 1) {
        const int hh = E.head_dim >> 1;
        const int pi0 = (fl % E.head_dim) >> 1;  // 8 consecutive pairs (16 | head_dim)
        float c[8], sn[8];
        if (rope_row) {
          const float4* cp = reinterpret_cast<const float4*>(rope_row + pi0);
          const float4* sp = reinterpret_cast<const float4*>(rope_row + hh + pi0);
          const float4 c0v = cp[0], c1v = cp[1], s0v = sp[0], s1v = sp[1];
          c[0] = c0v.x; c[1] = c0v.y; c[2] = c0v.z; c[3] = c0v.w; c[4] = c1v.x; c[5] = c1v.y; c[6] = c1v.z; c[7] = c1v.w;
          sn[0] = s0v.x; sn[1] = s0v.y; sn[2] = s0v.z; sn[3] = s0v.w; sn[4] = s1v.x; sn[5] = s1v.y; sn[6] = s1v.z; sn[7] = s1v.w;
        } else {
          const int pos = (int)min((long long)spos, E.rope_rows - 1);
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            c[i] = __ldg(E.rope_cos + (size_t)pos * hh + pi0 + i);
            sn[i] = __ldg(E.rope_sin + (size_t)pos * hh + pi0 + i);
          }
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const float x0 = v[2 * i], x1 = v[2 * i + 1];
          v[2 * i] = x0 * c[i] - x1 * sn[i];
          v[2 * i + 1] = x0 * sn[i] + x1 * c[i];
        }
      }
      store16<T>(reinterpret_cast<T*>(E.out[seg]) + srow * E.ld + fl, v);
      return;
    }
    case kEpiStoreT: {  // rows = output features, columns = tokens
      const int f = tile_m * BM + row;
      const int seg = f / E.seg_width;  // one segment per tile: seg_width is a multiple of 128
      const int fl = f - seg * E.seg_width;
      const int jb = tile_n * BN + c0;
      const bool rope = (E.rope_mask >> seg) & 1;
      // lane k of each warp finds the output row and RoPE position of token
      // jb + (k & 15) and the warp shares them: one round trip, not one per token
      const int kk = lane & 15;
      int my_pos = 0;
      const long long my_row = jb + kk < g.N ? column_target(E, jb + kk, &my_pos, g.status) : -1;
      my_pos = (int)min((long long)my_pos, E.rope_rows - 1);
      long long orow[16];
#pragma unroll
      for (int k = 0; k < 16; ++k) orow[k] = __shfl_sync(0xffffffffu, my_row, k);
      if (rope) {  // pair (2i, 2i+1) lives in lanes (l, l^1)
        const bool even = (fl & 1) == 0;
        const int hh = E.head_dim >> 1;
        const int pi = (fl % E.head_dim) >> 1;
        int pos[16];
#pragma unroll
        for (int k = 0; k < 16; ++k) pos[k] = __shfl_sync(0xffffffffu, my_pos, k);
        // all 16 table entries of each table: independent loads in flight together
        float cs[16], sn[16];
#pragma unroll
        for (int k = 0; k < 16; ++k) {
          cs[k] = __ldg(E.rope_cos + (size_t)pos[k] * hh + pi);
          sn[k] = __ldg(E.rope_sin + (size_t)pos[k] * hh + pi);
        }
#pragma unroll
        for (int k = 0; k < 16; ++k) {
          const float pv = __shfl_xor_sync(0xffffffffu, v[k], 1);
          if (jb + k < g.N) v[k] = even ? (v[k] * cs[k] - pv * sn[k]) : (pv * sn[k] + v[k] * cs[k]);
        }
      }
      if (f >= g.M) return;
      T* out = reinterpret_cast<T*>(E.out[seg]);
#pragma unroll
      for (int k = 0; k < 16; ++k)
        if (orow[k] >= 0) out[orow[k] * E.ld + fl] = from_f32<T>(v[k]);
      return;
    }
    case kEpiResidT: {
      const int f = tile_m * BM + row;
      if (f >= g.M) return;
      const int jb = tile_n * BN + c0;
      float* base = E.resid + (long long)jb * E.ld + f;
      // every load before any store, so the 16 reads are in flight together
      float r[16];
#pragma unroll
      for (int k = 0; k < 16; ++k) r[k] = jb + k < g.N ? __ldcg(base + (long long)k * E.ld) : 0.f;
#pragma unroll
      for (int k = 0; k < 16; ++k)
        if (jb + k < g.N) base[(long long)k * E.ld] = r[k] + v[k];
      return;
    }
    case kEpiSwigluT: {  // rows 0..63: gate g_f, rows 64..127: up u_f (same f)
      float* xbuf = reinterpret_cast<float*>(smem);  // [64][17]
      if (row >= 64) {
#pragma unroll
        for (int k = 0; k < 16; ++k) xbuf[(row - 64) * 17 + k] = v[k];
      }
      __syncthreads();
      if (row < 64) {
        const int f = tile_m * 64 + row;
        const int jb = tile_n * BN + c0;
        T* act = reinterpret_cast<T*>(E.out[0]);
        if (f < E.seg_width) {
#pragma unroll
          for (int k = 0; k < 16; ++k) {
            const int j = jb + k;
            if (j < g.N) {
              const float gv = v[k];
              const float u = xbuf[row * 17 + k];
              act[(long long)j * E.ld + f] = from_f32<T>(gv / (1.0f + expf(-gv)) * u);
            }
          }
        }
      }
      __syncthreads();
      return;
    }
    case kEpiLmHead: {  // rows = tokens, columns = vocabulary entries
      // Each thread owns one token and scans the tile's columns in increasing
      // order, chunk after chunk; its running max, first argmax and sum of
      // exp((z - max) * inv_temp) stay in a private shared-memory slot
      // between chunks, and the last chunk writes the tile's partials.
      float* st = reinterpret_cast<float*>(smem) + row * 4;
      const long long t = (long long)tile_m * BM + row;
      const long long V = g.N;
      const int jb = tile_n * BN + c0;
      const float it = E.inv_temp;
      float m = -INFINITY, sum = 0.f;
      int a = INT_MAX;
      if (c0 > 0) {
        m = st[0];
        sum = st[1];
        a = __float_as_int(st[2]);
      }
      if (t < g.M) {
        if (E.logsoftmax) {
          float* dst = E.logsoftmax + t * V + jb;
          if (jb + 16 <= V && ((V & 3) == 0)) {
#pragma unroll
            for (int i = 0; i < 4; ++i)
              reinterpret_cast<float4*>(dst)[i] =
                  make_float4(v[4 * i] * it, v[4 * i + 1] * it, v[4 * i + 2] * it, v[4 * i + 3] * it);
          } else {
#pragma unroll
            for (int k = 0; k < 16; ++k)
              if (jb + k < V) dst[k] = v[k] * it;
          }
        }
        // the chunk's maximum and first argmax in column order, then its
        // sum of exponentials (independent of one another), then one merge
        // with the running values (an earlier chunk keeps a tie)
        float cm = -INFINITY;
        int ca = INT_MAX;
#pragma unroll
        for (int k = 0; k < 16; ++k)
          if (jb + k < V && v[k] > cm) {
            cm = v[k];
            ca = jb + k;
          }
        if (cm != -INFINITY) {
          float cs = 0.f;
#pragma unroll
          for (int k = 0; k < 16; ++k)
            if (jb + k < V) cs += expf((v[k] - cm) * it);
          if (cm > m) {
            sum = (m == -INFINITY ? 0.f : sum * expf((m - cm) * it)) + cs;
            m = cm;
            a = ca;
          } else {
            sum += cs * expf((cm - m) * it);
          }
        }
      }
      if (c0 + 16 < BN) {
        st[0] = m;
        st[1] = sum;
        st[2] = __int_as_float(a);
      } else if (t < g.M) {
        const size_t o = (size_t)tile_n * g.M + t;
        E.part_max[o] = m;
        E.part_arg[o] = a;
        E.part_sum[o] = sum;
      }
      return;
    }
    case kEpiLmHeadT: {  // rows = vocabulary entries, columns = tokens
      // Per (tile, token): max, first argmax and sum of exp((z - max) * inv_temp)
      // over the tile's 128 rows.  The chunk goes through shared memory token-
      // major (row stride 136 floats: the 32 lanes of a read hit 32 banks);
      // eight threads per token scan 16 rows each in increasing order, then
      // merge (smaller index on ties).
      float* tv = reinterpret_cast<float*>(smem);  // [16 tokens][136]
      const long long V = g.M;
      const long long vr = (long long)tile_m * BM + row;
      const bool valid = vr < V;
      const int jb = tile_n * BN + c0;
      if (E.logsoftmax && valid) {
#pragma unroll
        for (int k = 0; k < 16; ++k)
          if (jb + k < g.N) E.logsoftmax[(long long)(jb + k) * V + vr] = v[k] * E.inv_temp;
      }
#pragma unroll
      for (int k = 0; k < 16; ++k) tv[k * 136 + row] = valid ? v[k] : -INFINITY;
      __syncthreads();
      const int k = row >> 3, part = row & 7;
      const float it = E.inv_temp;
      // this thread's 16 rows (increasing): maximum and first argmax, then
      // the sum of exponentials, independent of one another
      float xs[16];
      float m = -INFINITY, sum = 0.f;
      int a = INT_MAX;
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        xs[i] = tv[k * 136 + i * 8 + part];
        if (xs[i] > m) {
          m = xs[i];
          a = tile_m * BM + i * 8 + part;
        }
      }
      if (m != -INFINITY) {
#pragma unroll
        for (int i = 0; i < 16; ++i) sum += expf((xs[i] - m) * it);
      }
#pragma unroll
      for (int o = 1; o < 8; o <<= 1) {
        const float om = __shfl_xor_sync(0xffffffffu, m, o);
        const int oa = __shfl_xor_sync(0xffffffffu, a, o);
        const float os = __shfl_xor_sync(0xffffffffu, sum, o);
        const float nm = fmaxf(m, om);
        const float fs = m == -INFINITY ? 0.f : sum * expf((m - nm) * it);
        const float fo = om == -INFINITY ? 0.f : os * expf((om - nm) * it);
        if (om > m || (om == m && oa < a)) a = oa;
        m = nm;
        sum = fs + fo;
      }
      if (part == 0 && jb + k < g.N) {
        const size_t o = (size_t)tile_m * g.N + jb + k;
        E.part_max[o] = m;
        E.part_arg[o] = a;
        E.part_sum[o] = sum;
      }
      __syncthreads();
      return;
    }
  }
}

// Row-major epilogue with RoPE on the tile's segment: the RoPE table row of
// this thread's token (cos of the hd/2 pairs, then sin) goes into the
// drained stage memory with every copy in flight at once.  Rows are
// 2*(hd/2) + 4 floats apart, so eight threads reading 16 bytes each hit
// distinct bank groups.  Returns the row, or nullptr when nothing is staged.
template <int BN>
__device__ __forceinline__ const float* stage_rope_row(const GemmArgs& g, int tile_m, int tile_n, uint8_t* smem,
                                                       int spos) {
  const Epilogue& E = g.epi;
  if (E.kind != kEpiStore || E.head_dim > 128 || E.head_dim % 16) return nullptr;
  const int seg = (tile_n * BN) / E.seg_width;
  if (!((E.rope_mask >> seg) & 1)) return nullptr;
  const int hh = E.head_dim >> 1, stride = 2 * hh + 4;
  float* row = reinterpret_cast<float*>(smem) + threadIdx.x * stride;
  const long long t = (long long)tile_m * BM + threadIdx.x;
  if (t < g.M) {
    const int pos = (int)min((long long)spos, E.rope_rows - 1);
    const float* cs = E.rope_cos + (size_t)pos * hh;
    const float* sn = E.rope_sin + (size_t)pos * hh;
    for (int i = 0; i < hh; i += 4) {
      asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(row + i)), "l"(cs + i) : "memory");
      asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(row + hh + i)), "l"(sn + i) : "memory");
    }
  }
  asm volatile("cp.async.wait_all;" ::: "memory");
  return row;  // read back only by this thread
}

template <typename T, int BN>
__global__ void __launch_bounds__(128, 1) gemm_kernel(const __grid_constant__ GemmArgs g) {
  constexpr int STAGES = stages_for(BN);
  constexpr int BK = GT<T>::BK;
  constexpr int A_BYTES = BM * ROW_BYTES;
  constexpr int B_BYTES = BN * ROW_BYTES;
  constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  constexpr uint32_t TMEM_COLS = BN <= 32 ? 32 : (BN <= 64 ? 64 : (BN <= 128 ? 128 : 256));  // a power of two
  constexpr uint32_t IDESC = umma_idesc(BM, BN, GT<T>::FMT);

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  __shared__ __align__(8) uint64_t full_bar[STAGES];
  __shared__ __align__(8) uint64_t empty_bar[STAGES];
  __shared__ __align__(8) uint64_t acc_bar;
  __shared__ uint32_t tmem_slot;
  __shared__ volatile int abort_flag;
  __shared__ int cluster_abort;  // split-K, rank 0: some rank of the cluster gave up a wait

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  pdl_launch_dependents();
  const int tiles_m = (g.M + BM - 1) / BM;
  const int tiles_n = (g.N + BN - 1) / BN;
  int bid = blockIdx.x;
  const int split = bid % g.k_splits;
  bid /= g.k_splits;
  const int GN = g.group_n < 1 ? 1 : g.group_n;
  const int per_group = tiles_m * GN;
  const int grp = bid / per_group;
  const int rem = bid - grp * per_group;
  const int n0 = grp * GN;
  const int gw = min(GN, tiles_n - n0);
  const int tile_m = rem / gw;
  const int tile_n = n0 + rem % gw;

  const int num_kb = (g.K + BK - 1) / BK;
  const int kb_per = (num_kb + g.k_splits - 1) / g.k_splits;
  const int kb0 = split * kb_per;
  const int kb1 = min(num_kb, kb0 + kb_per);

  if (tid == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(smem_u32(&full_bar[s]), 1);
      mbar_init(smem_u32(&empty_bar[s]), 1);
    }
    mbar_init(smem_u32(&acc_bar), 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 2) tmem_alloc(smem_u32(&tmem_slot), TMEM_COLS);
  if (warp == 3 && lane == 0) {
    prefetch_tmap(&g.A.map[0]);
    prefetch_tmap(&g.B.map[0]);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_slot;

  if (!(warp == 0 && lane == 0)) pdl_wait();  // the producer waits after its weight prefetch
  if (warp == 0 && lane == 0) {
    // ------------------------------------------------ TMA producer
    auto load_a = [&](int st, int kb) {
      const uint32_t sa = smem_u32(smem + st * STAGE_BYTES);
      const CUtensorMap* map;
      int row;
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        operand_rows(g.A, tile_m * BM, h, tile_m, &map, &row);
        tma_load_2d(sa + h * (64 * ROW_BYTES), map, kb * BK, row, smem_u32(&full_bar[st]));
      }
    };
    auto load_b = [&](int st, int kb) {
      const CUtensorMap* map;
      int row;
      operand_rows(g.B, tile_n * BN, 0, tile_n, &map, &row);
      tma_load_2d(smem_u32(smem + st * STAGE_BYTES) + A_BYTES, map, kb * BK, row, smem_u32(&full_bar[st]));
    };
    // the first stages' weight operand is loaded while the previous kernel
    // may still run; the other operand only after pdl_wait()
    const int npre = g.pre_operand ? min(STAGES, kb1 - kb0) : 0;
    for (int i = 0; i < npre; ++i) {
      mbar_arrive_expect_tx(smem_u32(&full_bar[i]), STAGE_BYTES);
      if (g.pre_operand == 1) load_a(i, kb0 + i); else load_b(i, kb0 + i);
    }
    pdl_wait();
    for (int i = 0; i < npre; ++i) {
      if (g.pre_operand == 1) load_b(i, kb0 + i); else load_a(i, kb0 + i);
    }
    int s = npre % STAGES;
    uint32_t ph = npre == STAGES ? 1u : 0u;
    int issued = npre;
    for (int kb = kb0 + npre; kb < kb1; ++kb) {
      if (!mbar_wait(smem_u32(&empty_bar[s]), ph ^ 1, g.status)) { abort_flag = 1; break; }
      if (abort_flag) break;
      mbar_arrive_expect_tx(smem_u32(&full_bar[s]), STAGE_BYTES);
      load_a(s, kb);
      load_b(s, kb);
      ++issued;
      if (++s == STAGES) { s = 0; ph ^= 1; }
    }
    if (abort_flag) {
      // let copies already in flight land before shared memory is released
      int ss = s;
      uint32_t pp = ph;
      for (int i = 0; i < min(issued, STAGES); ++i) {
        if (--ss < 0) { ss = STAGES - 1; pp ^= 1; }
        mbar_wait(smem_u32(&full_bar[ss]), pp, nullptr);
      }
    }
  } else if (warp == 1 && lane == 0) {
    // ------------------------------------------------ MMA issuer
    int s = 0;
    uint32_t ph = 0;
    for (int kb = kb0; kb < kb1; ++kb) {
      if (!mbar_wait(smem_u32(&full_bar[s]), ph, g.status)) { abort_flag = 1; break; }
      if (abort_flag) break;
      tc_fence_after();
      const uint32_t sa = smem_u32(smem + s * STAGE_BYTES);
      const uint64_t ad = umma_desc_sw128(sa);
      const uint64_t bd = umma_desc_sw128(sa + A_BYTES);
#pragma unroll
      for (int k = 0; k < 4; ++k)  // 4 x 32 bytes of K per 128-byte row
        if (sizeof(T) == 2)
          mma_bf16(tmem, ad + 2 * k, bd + 2 * k, IDESC, (kb > kb0 || k > 0) ? 1u : 0u);
        else
          mma_tf32(tmem, ad + 2 * k, bd + 2 * k, IDESC, (kb > kb0 || k > 0) ? 1u : 0u);
      mma_commit(smem_u32(&empty_bar[s]));
      if (++s == STAGES) { s = 0; ph ^= 1; }
    }
    mma_commit(smem_u32(&acc_bar));  // also drains every MMA issued above
  }
  __syncwarp();

  // ------------------------------------------------------ epilogue
  if (!mbar_wait(smem_u32(&acc_bar), 0, g.status)) abort_flag = 1;
  tc_fence_after();
  __syncthreads();
  const bool aborted = abort_flag != 0;
  const uint32_t taddr = tmem + ((uint32_t)(warp * 32) << 16);
  int spos = 0;
  const long long srow = g.epi.kind == kEpiStore && (long long)tile_m * BM + tid < g.M
                             ? ctx_store_row(g.epi, (long long)tile_m * BM + tid, &spos, g.status)
                             : -1;
  if (!aborted && kb1 > kb0 && g.k_splits == 1) {
    const float* rope_row = BM * (2 * 64 + 4) * 4 <= STAGES * STAGE_BYTES
                                ? stage_rope_row<BN>(g, tile_m, tile_n, smem, spos)
                                : nullptr;
    if (BN >= 32) {
      // two chunks read from tensor memory per wait
#pragma unroll 1
      for (int c0 = 0; c0 < BN; c0 += 32) {
        float v[2][16];
        tmem_ld16x2(taddr + c0, v[0], taddr + c0 + 16, v[1]);
        epilogue_chunk<T, BN>(g, tile_m, tile_n, c0, v[0], smem, rope_row, srow, spos);
        epilogue_chunk<T, BN>(g, tile_m, tile_n, c0 + 16, v[1], smem, rope_row, srow, spos);
      }
    } else {
      float v[16];
      tmem_ld16(taddr, v);
      epilogue_chunk<T, BN>(g, tile_m, tile_n, 0, v, smem, rope_row, srow, spos);
    }
  }
  if (g.k_splits > 1) {
    // every rank: accumulator -> own shared memory [128 rows][BN] (all MMAs
    // and copies have completed, so the stage memory is free)
    float* part = reinterpret_cast<float*>(smem + kPartialOffset);
    if (!aborted && kb1 > kb0) {
#pragma unroll 1
      for (int c0 = 0; c0 < BN; c0 += 16) {
        float v[16];
        tmem_ld16(taddr + c0, v);
        float4* p = reinterpret_cast<float4*>(part + tid * BN + c0);
#pragma unroll
        for (int i = 0; i < 4; ++i) p[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
      }
    } else {
      for (int c = 0; c < BN; ++c) part[tid * BN + c] = 0.f;
    }
    cluster_sync_all();  // every rank's partial tile and abort flag are visible to the cluster
    // a rank that gave up a wait left zeros as its partial: rank 0 then skips
    // the store (the device status word already records the failure)
    if (cluster_rank() == 0 && tid == 0) {
      int any = 0;
      for (int u = 0; u < g.k_splits; ++u) any |= ld_dsmem_s32(map_rank(smem_u32((const void*)&abort_flag), (uint32_t)u));
      cluster_abort = any;
    }
    // Every rank sums a slice of the tile's rows over all ranks (one float4
    // column per thread and round, every source in flight at once, summed in
    // rank order) and writes the result over rank 0's partial of that slice:
    // the slice is read and written by this rank only.
    if (BN <= 128) {
      const int k = g.k_splits;
      const uint32_t rank = cluster_rank();
      const int rpr = (BM + k - 1) / k;  // rows per rank
      const int row0 = (int)rank * rpr, nrow = max(0, min(BM, row0 + rpr) - row0);
      constexpr int C4 = BN / 4;
      const uint32_t part_base = smem_u32(part);
      const uint32_t red_base = map_rank(part_base, 0u);
      for (int it = tid; it < nrow * C4; it += 128) {
        const int r = row0 + it / C4, c4 = it - (it / C4) * C4;
        const uint32_t off = (uint32_t)((r * BN + c4 * 4) * 4);
        float4 q[16];
#pragma unroll
        for (int u = 0; u < 16; ++u)
          if (u < k) q[u] = ld_dsmem_v4(map_rank(part_base + off, (uint32_t)u));
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int u = 0; u < 16; ++u)
          if (u < k) {
            acc.x += q[u].x;
            acc.y += q[u].y;
            acc.z += q[u].z;
            acc.w += q[u].w;
          }
        asm volatile("st.shared::cluster.v4.f32 [%0], {%1,%2,%3,%4};" ::"r"(red_base + off), "f"(acc.x),
                     "f"(acc.y), "f"(acc.z), "f"(acc.w)
                     : "memory");
      }
    }
    cluster_sync_all();  // rank 0's tile holds the sums; no rank reads another's memory any more
    if (cluster_rank() == 0 && !cluster_abort) {
      const float* red = part;
#pragma unroll 1
      for (int c0 = 0; c0 < BN; c0 += 16) {
        float v[16];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const float4 q = *reinterpret_cast<const float4*>(red + tid * BN + c0 + 4 * i);
          v[4 * i] = q.x;
          v[4 * i + 1] = q.y;
          v[4 * i + 2] = q.z;
          v[4 * i + 3] = q.w;
        }
        epilogue_chunk<T, BN>(g, tile_m, tile_n, c0, v, smem, nullptr, srow, spos);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

// ---------------------------------------------------------------------------
// 2-SM tile (cta_group::2) for the row-major store GEMMs (kEpiStore, bf16):
// a cluster of two CTAs computes a 256 x 256 tile.  Rank r loads rows
// [256 i + 128 r, +128) of A and rows [256 j + 128 r, +128) of B into its own
// shared memory, 32 KB per 64-deep stage; rank 0 issues
// tcgen05.mma.cta_group::2 with M = 256, N = 256, whose operands are read from
// both CTAs and whose accumulator rows land in the tensor memory of the CTA
// that holds them.  Per SM that is 32 KB of operands per 128 x 256 x 64 of
// MMA work instead of 48 KB, so the same bytes in flight feed 1.5x the
// tensor-core work.  Both CTAs' loads are counted on rank 0's full barrier
// (armed by rank 0 for the pair's 64 KB); rank 0's commits arrive on the
// empty and accumulator barriers of both CTAs.  Three stages per CTA and two
// CTAs per SM.  Each output element is one K-ordered chain of MMAs, as in
// gemm_kernel.
constexpr int kPairStages = 3;
constexpr int kPairStageBytes = 2 * BM * ROW_BYTES;  // A half + B half
constexpr int kPairSmem = kPairStages * kPairStageBytes + 1024;
static_assert(BM * (2 * 64 + 4) * 4 <= kPairStages * kPairStageBytes, "RoPE rows fit the drained stages");

__global__ void __launch_bounds__(128, 1) gemm_pair_kernel(const __grid_constant__ GemmArgs g) {
  constexpr int BN = 256;
  constexpr int STAGES = kPairStages;
  constexpr int BK = 64;
  constexpr int A_BYTES = BM * ROW_BYTES;
  constexpr int STAGE_BYTES = kPairStageBytes;
  constexpr uint32_t TMEM_COLS = 256;
  constexpr uint32_t IDESC = umma_idesc(2 * BM, BN, 1);

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  __shared__ __align__(8) uint64_t full_bar[STAGES];
  __shared__ __align__(8) uint64_t empty_bar[STAGES];
  __shared__ __align__(8) uint64_t acc_bar;
  __shared__ uint32_t tmem_slot;
  __shared__ volatile int abort_flag;
  __shared__ int pair_abort;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  pdl_launch_dependents();
  const uint32_t rank = cluster_rank();
  const bool leader = rank == 0;
  const int tiles_m = (g.M + 2 * BM - 1) / (2 * BM);
  const int tiles_n = (g.N + BN - 1) / BN;
  const int bid = blockIdx.x >> 1;
  const int GN = g.group_n < 1 ? 1 : g.group_n;
  const int per_group = tiles_m * GN;
  const int grp = bid / per_group;
  const int rem = bid - grp * per_group;
  const int n0 = grp * GN;
  const int gw = min(GN, tiles_n - n0);
  const int tile_m = rem / gw;          // 256-row tile of the pair
  const int tile_n = n0 + rem % gw;     // 256-column tile
  const int my_m = tile_m * 2 + (int)rank;  // this CTA's 128-row tile
  const int num_kb = (g.K + BK - 1) / BK;

  if (tid == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(smem_u32(&full_bar[s]), 1);
      mbar_init(smem_u32(&empty_bar[s]), 1);
    }
    mbar_init(smem_u32(&acc_bar), 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 2) tmem_alloc_pair(smem_u32(&tmem_slot), TMEM_COLS);
  if (warp == 3 && lane == 0) {
    prefetch_tmap(&g.A.map[0]);
    prefetch_tmap(&g.B.map[0]);
  }
  tc_fence_before();
  cluster_sync_all();  // both CTAs' barriers and tensor memory exist before either touches the other's
  tc_fence_after();
  const uint32_t tmem = tmem_slot;

  // This thread's output row, RoPE position and (head_dim 128, RoPE tiles)
  // the 64 cos and 64 sin entries of that position, loaded into registers
  // while the mainloop runs, so the epilogue waits on no global load.
  const Epilogue& E = g.epi;
  const long long t = (long long)my_m * BM + tid;
  const int seg_t = (tile_n * BN) / E.seg_width;
  const bool rope_regs = E.kind == kEpiStore && E.head_dim == 128 && ((E.rope_mask >> seg_t) & 1) &&
                         (E.seg_width % BN) == 0;
  int spos = 0;
  long long srow = -1;
  float4 rc[16], rs[16];
  auto row_prefetch = [&]() {
    srow = t < g.M ? ctx_store_row(E, t, &spos, g.status) : -1;
    if (rope_regs && srow >= 0) {
      const int pos = (int)min((long long)spos, E.rope_rows - 1);
      const float4* cp = reinterpret_cast<const float4*>(E.rope_cos + (size_t)pos * 64);
      const float4* sp = reinterpret_cast<const float4*>(E.rope_sin + (size_t)pos * 64);
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        rc[i] = __ldg(cp + i);
        rs[i] = __ldg(sp + i);
      }
    }
  };
  if (!(warp == 0 && lane == 0)) {
    pdl_wait();  // the producer waits after its weight prefetch
    row_prefetch();
  }
  if (warp == 0 && lane == 0) {
    // ------------------------------------------------ TMA producer (both CTAs)
    auto full_of = [&](int st) { return map_rank(smem_u32(&full_bar[st]), 0u); };
    auto load_a = [&](int st, int kb) {
      const uint32_t sa = smem_u32(smem + st * STAGE_BYTES);
      const CUtensorMap* map;
      int row;
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        operand_rows(g.A, my_m * BM, h, my_m, &map, &row);
        tma_load_2d_pair(sa + h * (64 * ROW_BYTES), map, kb * BK, row, full_of(st));
      }
    };
    auto load_b = [&](int st, int kb) {
      const CUtensorMap* map;
      int row;
      operand_rows(g.B, tile_n * BN + (int)rank * BM, 0, tile_n, &map, &row);
      tma_load_2d_pair(smem_u32(smem + st * STAGE_BYTES) + A_BYTES, map, kb * BK, row, full_of(st));
    };
    // rank 0 arms each stage for the bytes of both CTAs; the peer's copies
    // may land before that (the transaction count then dips below zero, but
    // the phase cannot complete before rank 0's arrival)
    const int npre = g.pre_operand ? min(STAGES, num_kb) : 0;
    for (int i = 0; i < npre; ++i) {
      if (leader) mbar_arrive_expect_tx(smem_u32(&full_bar[i]), 2 * STAGE_BYTES);
      if (g.pre_operand == 1) load_a(i, i); else load_b(i, i);
    }
    pdl_wait();
    for (int i = 0; i < npre; ++i) {
      if (g.pre_operand == 1) load_b(i, i); else load_a(i, i);
    }
    int s = npre % STAGES;
    uint32_t ph = npre == STAGES ? 1u : 0u;
    int issued = npre;
    for (int kb = npre; kb < num_kb; ++kb) {
      if (!mbar_wait(smem_u32(&empty_bar[s]), ph ^ 1, g.status)) { abort_flag = 1; break; }
      if (abort_flag) break;
      if (leader) mbar_arrive_expect_tx(smem_u32(&full_bar[s]), 2 * STAGE_BYTES);
      load_a(s, kb);
      load_b(s, kb);
      ++issued;
      if (++s == STAGES) { s = 0; ph ^= 1; }
    }
    if (abort_flag && leader) {
      // copies already in flight (both CTAs' copies of every armed stage)
      // land before shared memory is released
      int ss = s;
      uint32_t pp = ph;
      for (int i = 0; i < min(issued, STAGES); ++i) {
        if (--ss < 0) { ss = STAGES - 1; pp ^= 1; }
        mbar_wait(smem_u32(&full_bar[ss]), pp, nullptr);
      }
    }
    row_prefetch();  // the last loads are issued a few stages before the mainloop ends
  } else if (warp == 1 && lane == 0 && leader) {
    // ------------------------------------------------ MMA issuer (rank 0)
    int s = 0;
    uint32_t ph = 0;
    for (int kb = 0; kb < num_kb; ++kb) {
      if (!mbar_wait(smem_u32(&full_bar[s]), ph, g.status)) { abort_flag = 1; break; }
      if (abort_flag) break;
      tc_fence_after();
      const uint32_t sa = smem_u32(smem + s * STAGE_BYTES);
      const uint64_t ad = umma_desc_sw128(sa);
      const uint64_t bd = umma_desc_sw128(sa + A_BYTES);
#pragma unroll
      for (int k = 0; k < 4; ++k)  // 4 x 32 bytes of K per 128-byte row
        mma_bf16_pair(tmem, ad + 2 * k, bd + 2 * k, IDESC, (kb > 0 || k > 0) ? 1u : 0u);
      mma_commit_pair(smem_u32(&empty_bar[s]), (uint16_t)0x3);
      if (++s == STAGES) { s = 0; ph ^= 1; }
    }
    mma_commit_pair(smem_u32(&acc_bar), (uint16_t)0x3);  // also drains every MMA issued above
  }
  __syncwarp();

  // ------------------------------------------------------ epilogue
  if (!mbar_wait(smem_u32(&acc_bar), 0, g.status)) abort_flag = 1;
  tc_fence_after();
  __syncthreads();
  cluster_sync_all();  // both CTAs' abort flags are final and visible
  if (tid == 0)
    pair_abort = abort_flag | ld_dsmem_s32(map_rank(smem_u32((const void*)&abort_flag), rank ^ 1u));
  __syncthreads();
  const uint32_t taddr = tmem + ((uint32_t)(warp * 32) << 16);
  const bool seg_rope = (E.rope_mask >> seg_t) & 1;
  const bool tma_out = E.kind == kEpiStore && E.out_tma && (E.pos_mode == 0 || E.pos_mode == 1) &&
                       (E.seg_width % BN) == 0 && seg_t < 2 && (rope_regs || !seg_rope);
  if (!pair_abort && num_kb > 0 && tma_out) {
    // The tile goes through the drained stage memory as four 128-row x 64-
    // column boxes in the output map's 128-byte swizzle (16-byte chunk j of
    // row r at chunk j ^ (r & 7): a warp's 32 rows hit all banks), then out
    // by four TMA stores: whole lines instead of one 32-byte piece per row
    // and column chunk.  Chunks c and c + 8 (the same RoPE pairs of the
    // tile's two heads) come from tensor memory together.
    const int fl0 = tile_n * BN - seg_t * E.seg_width;
    uint8_t* tile_smem = smem;  // 4 x 16 KB, 1024-byte aligned
#pragma unroll
    for (int c = 0; c < 8; ++c) {
      float v[2][16];
      tmem_ld16x2(taddr + 16 * c, v[0], taddr + 16 * (c + 8), v[1]);
      if (rope_regs) {
        const float4 c0v = rc[2 * c], c1v = rc[2 * c + 1];
        const float4 s0v = rs[2 * c], s1v = rs[2 * c + 1];
        const float cs[8] = {c0v.x, c0v.y, c0v.z, c0v.w, c1v.x, c1v.y, c1v.z, c1v.w};
        const float sn[8] = {s0v.x, s0v.y, s0v.z, s0v.w, s1v.x, s1v.y, s1v.z, s1v.w};
#pragma unroll
        for (int hd = 0; hd < 2; ++hd)
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const float x0 = v[hd][2 * i], x1 = v[hd][2 * i + 1];
            v[hd][2 * i] = x0 * cs[i] - x1 * sn[i];
            v[hd][2 * i + 1] = x0 * sn[i] + x1 * cs[i];
          }
      }
#pragma unroll
      for (int hd = 0; hd < 2; ++hd) {
        const int cc = c + 8 * hd;  // 16-column chunk of the tile
        uint8_t* box = tile_smem + (cc >> 2) * (BM * ROW_BYTES);
        const int j0 = (cc & 3) * 2;
        uint8_t* rowp = box + tid * ROW_BYTES;
        *reinterpret_cast<uint4*>(rowp + ((j0 ^ (tid & 7)) << 4)) = V16<__nv_bfloat16>::pack(v[hd]);
        *reinterpret_cast<uint4*>(rowp + (((j0 + 1) ^ (tid & 7)) << 4)) = V16<__nv_bfloat16>::pack(v[hd] + 8);
      }
    }
    fence_proxy_async();
    __syncthreads();
    if (tid == 0) {
#pragma unroll
      for (int b = 0; b < BN / 64; ++b)
        tma_store_2d(&E.out_map[seg_t], smem_u32(tile_smem + b * (BM * ROW_BYTES)), fl0 + 64 * b, my_m * BM);
      tma_store_commit();
      tma_store_wait_all();
    }
  } else if (!pair_abort && num_kb > 0 && rope_regs) {
    // the tile is one segment and two whole heads: chunk c holds pairs
    // 8 (c % 8) .. 8 (c % 8) + 7 of its head
    const int col_t = tile_n * BN;
    const int fl0 = col_t - seg_t * E.seg_width;
    __nv_bfloat16* out = reinterpret_cast<__nv_bfloat16*>(E.out[seg_t]);
    // chunks c and c + 8 (the same pairs of the tile's two heads) are read
    // from tensor memory together: one wait for both
#pragma unroll
    for (int c = 0; c < 8; ++c) {
      float v[2][16];
      tmem_ld16x2(taddr + 16 * c, v[0], taddr + 16 * (c + 8), v[1]);
      const float4 c0v = rc[2 * c], c1v = rc[2 * c + 1];
      const float4 s0v = rs[2 * c], s1v = rs[2 * c + 1];
      const float cs[8] = {c0v.x, c0v.y, c0v.z, c0v.w, c1v.x, c1v.y, c1v.z, c1v.w};
      const float sn[8] = {s0v.x, s0v.y, s0v.z, s0v.w, s1v.x, s1v.y, s1v.z, s1v.w};
#pragma unroll
      for (int hd = 0; hd < 2; ++hd) {
        const int cc = c + 8 * hd;
        if (srow >= 0 && col_t + 16 * cc < g.N) {
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const float x0 = v[hd][2 * i], x1 = v[hd][2 * i + 1];
            v[hd][2 * i] = x0 * cs[i] - x1 * sn[i];
            v[hd][2 * i + 1] = x0 * sn[i] + x1 * cs[i];
          }
          store16<__nv_bfloat16>(out + srow * E.ld + fl0 + 16 * cc, v[hd]);
        }
      }
    }
  } else if (!pair_abort && num_kb > 0) {
    const float* rope_row = stage_rope_row<BN>(g, my_m, tile_n, smem, spos);
#pragma unroll 1
    for (int c0 = 0; c0 < BN; c0 += 32) {
      float v[2][16];
      tmem_ld16x2(taddr + c0, v[0], taddr + c0 + 16, v[1]);
      epilogue_chunk<__nv_bfloat16, BN>(g, my_m, tile_n, c0, v[0], smem, rope_row, srow, spos);
      epilogue_chunk<__nv_bfloat16, BN>(g, my_m, tile_n, c0 + 16, v[1], smem, rope_row, srow, spos);
    }
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // neither CTA frees the pair's tensor memory while the other still reads it
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, TMEM_COLS);
  }
}

cudaError_t prepare_pair() { return ensure_smem_limit((const void*)gemm_pair_kernel, kPairSmem); }

cudaError_t launch_pair(const GemmArgs& g, cudaStream_t s) {
  cudaError_t e;
  if ((e = prepare_pair()) != cudaSuccess) return e;
  if (g.dtype != HDF_BF16 || g.k_splits != 1 || g.bn != 256 || g.epi.kind != kEpiStore) return cudaErrorInvalidValue;
  const long long tiles = (long long)((g.M + 2 * BM - 1) / (2 * BM)) * ((g.N + 255) / 256);
  return launch_kernel(gemm_pair_kernel, dim3((unsigned)(2 * tiles)), dim3(128), (size_t)kPairSmem, s, 2u, g);
}

// Function attributes of one instantiation on the current device: the
// dynamic shared memory and clusters of up to 16 CTAs.
template <typename T, int BN>
cudaError_t prepare_bn() {
  return ensure_smem_limit((const void*)gemm_kernel<T, BN>, (size_t)smem_for(BN), true);
}

template <typename T, int BN>
cudaError_t launch_bn(const GemmArgs& g, cudaStream_t s) {
  cudaError_t e;
  if ((e = prepare_bn<T, BN>()) != cudaSuccess) return e;
  if (g.k_splits < 1 || g.k_splits > 16 || (g.k_splits > 1 && BN > 128)) return cudaErrorInvalidValue;
  const long long tiles = (long long)((g.M + BM - 1) / BM) * ((g.N + BN - 1) / BN) * g.k_splits;
  // the splits of one tile are consecutive blocks: one cluster
  return launch_kernel(gemm_kernel<T, BN>, dim3((unsigned)tiles), dim3(128), (size_t)smem_for(BN), s,
                       (unsigned)g.k_splits, g);
}

// CTAs resident at once when the grid is made of clusters of `cluster` CTAs
// (the occupancy API packs clusters into GPCs); -1 if it cannot be asked.
template <typename T, int BN>
int resident_ctas_bn(int cluster) {
  int n = 0;
  if (prepare_bn<T, BN>() != cudaSuccess ||
      max_active_clusters((const void*)gemm_kernel<T, BN>, 128, (size_t)smem_for(BN), cluster, &n) != cudaSuccess ||
      n <= 0) {
    cudaGetLastError();
    return -1;
  }
  return n * cluster;
}

template <typename T>
int resident_ctas_t(int bn, int cluster) {
  switch (bn) {
    case 16: return resident_ctas_bn<T, 16>(cluster);
    case 32: return resident_ctas_bn<T, 32>(cluster);
    case 64: return resident_ctas_bn<T, 64>(cluster);
    case 128: return resident_ctas_bn<T, 128>(cluster);
    case 224: return resident_ctas_bn<T, 224>(cluster);
    case 256: return resident_ctas_bn<T, 256>(cluster);
    default: return -1;
  }
}

template <typename T>
cudaError_t launch_t(const GemmArgs& g, cudaStream_t s) {
  switch (g.bn) {
    case 16: return launch_bn<T, 16>(g, s);
    case 32: return launch_bn<T, 32>(g, s);
    case 64: return launch_bn<T, 64>(g, s);
    case 128: return launch_bn<T, 128>(g, s);
    case 224: return launch_bn<T, 224>(g, s);
    case 256: return launch_bn<T, 256>(g, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

int gemm_stages(int, int bn) { return stages_for(bn); }

int gemm_resident_ctas(int dtype, int bn, int cluster) {
  if (cluster < 1 || cluster > 16) return -1;
  const int bi = bn == 16 ? 0 : bn == 32 ? 1 : bn == 64 ? 2 : bn == 128 ? 3 : bn == 256 ? 4 : bn == 224 ? 5 : -1;
  if (bi < 0) return -1;
  // the occupancy answer is cached per device by max_active_clusters
  return dtype == HDF_BF16 ? resident_ctas_t<__nv_bfloat16>(bn, cluster) : resident_ctas_t<float>(bn, cluster);
}
size_t gemm_smem_bytes(int, int bn) { return (size_t)smem_for(bn); }

cudaError_t launch_gemm(const GemmArgs& g, cudaStream_t s) {
  if (g.M <= 0 || g.N <= 0) return cudaSuccess;
  if (g.pair) return launch_pair(g, s);
  return g.dtype == HDF_BF16 ? launch_t<__nv_bfloat16>(g, s) : launch_t<float>(g, s);
}

}  // namespace hdf
