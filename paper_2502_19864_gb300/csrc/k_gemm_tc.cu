// k_gemm_tc.cu -- tcgen05 / TMEM / TMA GEMM for sm_103a with the step's fused epilogues.
//
// C[M, N] = A[M, K] B[N, K]^T, bf16 operands (both K-major), fp32 accumulation in TMEM.
// This carries every frozen-weight GEMM of the forward (QKV, attention output, FFN up with
// the bias+GELU or SwiGLU epilogue, FFN down) and every transposed-weight dX GEMM of the
// backward (fused GELU' / SwiGLU' / residual epilogues) -- the dense contractions of the
// step.
//
// Structure (one persistent CTA per SM, 320 threads):
//   warp 0      TMA producer: 128 x 64 A tiles and BN x 64 B tiles (BN = 128, 192 or 256;
//               128-byte swizzle) into a STAGES-deep shared-memory ring, completion tracked
//               by mbarrier tx counts;
//   warp 1      allocates 2*BN TMEM columns (two accumulators); one thread issues
//               tcgen05.mma (M = 128, N = BN, K = 16) and tcgen05.commit to free each stage
//               and to publish each finished accumulator;
//   warps 2..9  epilogue: two warps per TMEM lane quadrant (warp w may only read lanes
//               32 * (w % 4) .. + 31), each taking half of the tile's columns: tcgen05.ld,
//               fused math, then each 32 x 32 output chunk is staged in shared memory
//               (TMA swizzle layout, conflict-free) and written by a TMA tensor store, which
//               coalesces the rows and clips ragged edges; the second accumulator lets the
//               next tile's main loop overlap this.
// Every mbarrier wait is bounded (global timer); on expiry the kernel records
// RA_DEVERR_TIMEOUT, drains its own copies and MMAs, frees TMEM and returns.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstring>
#include <mutex>
#include <unordered_map>

#include "common.cuh"
#include "kernels.h"
#include "tcgen05.cuh"

namespace ra {
namespace {

using namespace tc;

constexpr int BM = 128, BK = 64;

// epilogue staging: 4 KB per warp, one 32 x 32 f32 chunk or two 32 x 32 bf16 chunks (then
// a second store can be staged while the first is still being read); this keeps the full
// operand ring (224 KB in all)
constexpr int SLOT_BYTES = 4096, NSLOT = 1;

// epilogues that read a saved operand per output element (GELU', residual, SwiGLU')
template <int EPI>
struct EpiTraits {
  // the GELU epilogues evaluate erf per element: 12 epilogue warps (three per TMEM lane
  // quadrant) for them, 8 for the others
  static constexpr int WARPS = (EPI == EPI_BIAS_GELU || EPI == EPI_BIAS_GELU_G) ? 12 : 8;
  static constexpr int THREADS = (2 + WARPS) * 32;
  static constexpr bool AUX = EPI == EPI_MUL || EPI == EPI_RESID || EPI == EPI_DSWIGLU;
  // stream-K partial and finisher units (the plain store epilogue only)
  static constexpr bool SK = EPI == EPI_STORE;
};

// Every epilogue stages through 4 KB per warp, which keeps the full operand ring.  AUX
// epilogues TMA-load their operand chunk into that area: bf16 factor operands use two 2 KB
// regions (the next chunk loads while this one computes); 4 KB operands (fp32 residual,
// packed gate|up) use one region, whose first chunk per tile loads during the main loop.
template <int BN, bool AUX, int EW = 8>
struct TileCfg {
  // the operand ring gives up a stage to the staging of the extra epilogue warps (a
  // 192-wide ring keeps 4 stages either way: 40 KB stages)
  static constexpr int STAGES = BN == 256 ? (EW > 8 ? 3 : 4) : BN == 192 ? 4 : (EW > 8 ? 5 : 6);
  static constexpr int A_BYTES = BM * BK * 2;
  static constexpr int B_BYTES = BN * BK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  // two accumulators of BN columns; the allocation is a power of two
  static constexpr int TMEM_COLS = 2 * BN <= 256 ? 256 : 512;
  static constexpr int WARP_STAGING = NSLOT * SLOT_BYTES;
  static constexpr int STAGING = EW * WARP_STAGING;
  static constexpr int SMEM = STAGES * STAGE_BYTES + STAGING + 1024;  // + alignment slack
};

struct TcParams {
  int M, N, K;
  // B stored [K, N], read MN-major: 1 = BN / 64 TMA boxes of 64 x 64 per stage; 2 = one
  // box of a 3-D view (64 columns, K rows, N / 64 column blocks) that lands as the same
  // BN / 64 swizzle atoms (N a multiple of 64)
  int b_kn;
  int n_tiles_n, m_tiles, num_tiles, k_blocks;
  int epi;
  void* C; int ldc; int c_dtype;
  const float* bias;
  void* C2; int ldc2; int c2_dtype;
  const void* aux; int ldaux; int aux_dtype;
  unsigned* err;
  // stream-K (sk_iters > 0): tiles [0, dp_tiles) go one per CTA and round; the k-blocks of
  // the tiles after them, numbered tile by tile, are split evenly over CTAs 0 .. sk_ctas - 1
  int dp_tiles, sk_ctas, sk_iters;
  float* sk_ws;         // one partial accumulator slot (SK_SLOT_FLOATS) per CTA
  unsigned* sk_flags;   // per (CTA, epilogue warp): 1 while that warp's partial is published
};

// A partial accumulator slot holds a whole 128 x 256 tile in fp32: for output column chunk
// c (32 columns) and column group q (4 columns), the 128 rows' float4s are contiguous, so a
// warp moves 512 consecutive bytes per access.
constexpr int SK_SLOT_FLOATS = BM * 256;
constexpr int SK_MAX_WARPS = 12;

// One CTA's work as an ordered list of units (tile, k-blocks [kb0, kb1), kind):
//   kind 0  a whole tile;
//   kind 1  partial: the accumulator of k-blocks [kb0, kb1) of a stream-K tile goes to this
//           CTA's slot; a CTA with a higher index finishes the tile;
//   kind 2  finisher: the last k-blocks of a stream-K tile; the epilogue first adds the
//           partials of the lower-indexed CTAs that did the tile's first k-blocks, in
//           ascending CTA order (a fixed order: the result does not depend on timing).
// Order within a CTA: the partial first, so that a finisher only ever waits for work its
// source CTAs do before anything else (and sources have lower indexes, so they were
// dispatched first); then the finisher, whose wait for the partials and whose reads of them
// then overlap the main loops of the tiles that follow; then the whole stream-K tiles and
// the data-parallel tiles.
struct Sched {
  int c, K, stride, dp_tiles, n_dp, n_p, n_mid, n_fin, t_first, t_last, b, e;
  __device__ void init(const TcParams& p, int cta, int grid) {
    c = cta; K = p.k_blocks; stride = grid; dp_tiles = p.dp_tiles;
    n_dp = dp_tiles > c ? (dp_tiles - c + grid - 1) / grid : 0;
    n_p = n_mid = n_fin = 0;
    t_first = 0; t_last = -1; b = e = 0;
    if (p.sk_iters > 0 && c < p.sk_ctas) {
      b = (int)((long long)c * p.sk_iters / p.sk_ctas);
      e = (int)((long long)(c + 1) * p.sk_iters / p.sk_ctas);
      if (b < e) {
        t_first = b / K;
        t_last = (e - 1) / K;
        n_fin = (b % K != 0 && (t_first + 1) * K <= e) ? 1 : 0;
        n_p = e % K != 0 ? 1 : 0;
        n_mid = t_last - t_first + 1 - n_p - n_fin;
      }
    }
  }
  __device__ int count() const { return n_p + n_dp + n_mid + n_fin; }
  __device__ void unit(int u, int& tile, int& kb0, int& kb1, int& kind) const {
    if (u < n_p) {
      const int base = t_last * K;
      tile = dp_tiles + t_last; kb0 = max(b, base) - base; kb1 = e - base; kind = 1;
      return;
    }
    u -= n_p;
    if (u < n_fin) {
      tile = dp_tiles + t_first; kb0 = b - t_first * K; kb1 = K; kind = 2;
      return;
    }
    u -= n_fin;
    if (u < n_mid) {  // whole tiles
      tile = dp_tiles + t_first + n_fin + u; kb0 = 0; kb1 = K; kind = 0;
      return;
    }
    u -= n_mid;
    tile = c + u * stride; kb0 = 0; kb1 = K; kind = 0;
  }
  // first CTA that holds k-blocks of stream-K tile t: the owner of its first iteration,
  // the largest cc with floor(cc * I / G) <= t * K
  __device__ static int first_source(const TcParams& p, int t) {
    const long long i = (long long)t * p.k_blocks;
    return (int)(((i + 1) * p.sk_ctas - 1) / p.sk_iters);
  }
};

// ---- TMA and bulk-copy helpers ------------------------------------------------------------
__device__ __forceinline__ void tma_load_2d(const CUtensorMap* tm, uint32_t dst, uint64_t* bar,
                                            int c0, int c1) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tm)), "r"(c0), "r"(c1), "r"(smem_u32(bar))
      : "memory");
}
__device__ __forceinline__ void tma_load_3d(const CUtensorMap* tm, uint32_t dst, uint64_t* bar,
                                            int c0, int c1, int c2) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tm)), "r"(c0), "r"(c1), "r"(c2), "r"(smem_u32(bar))
      : "memory");
}
__device__ __forceinline__ void tma_store_2d(const CUtensorMap* tm, uint32_t src, int c0, int c1) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];" ::"l"(
                   reinterpret_cast<uint64_t>(tm)),
               "r"(c0), "r"(c1), "r"(src)
               : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// at most N bulk stores of this thread may still be reading shared memory
template <int N>
__device__ __forceinline__ void bulk_wait_read() {
  asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
// ---- epilogue ---------------------------------------------------------------------------------
__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}
// Writes this thread's row (lane) of a 32 x 32 chunk into a staging slot in the TMA swizzle
// layout the store map uses: bf16 rows are 64 B under the 64-byte swizzle (16-byte chunk q
// of row r at q ^ ((r >> 1) & 3)), f32 rows 128 B under the 128-byte swizzle (q ^ (r & 7)).
// Lanes 0..7 then hit eight different bank groups for every q: no bank conflicts.
// (Output chunks use stage_half for f32; the 128-byte form serves the f32 operand staging.)
__device__ __forceinline__ void stage_row(uint8_t* slot, int dt, int lane, const float* x) {
  if (dt == DT_BF16) {
    uint8_t* row = slot + lane * 64;
    const int sw = (lane >> 1) & 3;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      uint4 v;
      v.x = pack_bf16x2(x[8 * q + 0], x[8 * q + 1]);
      v.y = pack_bf16x2(x[8 * q + 2], x[8 * q + 3]);
      v.z = pack_bf16x2(x[8 * q + 4], x[8 * q + 5]);
      v.w = pack_bf16x2(x[8 * q + 6], x[8 * q + 7]);
      *reinterpret_cast<uint4*>(row + ((q ^ sw) << 4)) = v;
    }
  } else {
    uint8_t* row = slot + lane * 128;
    const int sw = lane & 7;
#pragma unroll
    for (int q = 0; q < 8; ++q)
      *reinterpret_cast<float4*>(row + ((q ^ sw) << 4)) =
          make_float4(x[4 * q], x[4 * q + 1], x[4 * q + 2], x[4 * q + 3]);
  }
}

// Reads this thread's row (lane) of a 32 x 32 chunk from the TMA swizzle layout (inverse of
// stage_row).
__device__ __forceinline__ void unstage_row(const uint8_t* slot, int dt, int lane, float* x) {
  if (dt == DT_BF16) {
    const uint8_t* row = slot + lane * 64;
    const int sw = (lane >> 1) & 3;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const uint4 v = *reinterpret_cast<const uint4*>(row + ((q ^ sw) << 4));
      const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float2 f = __bfloat1622float2(h[i]);
        x[8 * q + 2 * i] = f.x;
        x[8 * q + 2 * i + 1] = f.y;
      }
    }
  } else {
    const uint8_t* row = slot + lane * 128;
    const int sw = lane & 7;
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const float4 v = *reinterpret_cast<const float4*>(row + ((q ^ sw) << 4));
      x[4 * q] = v.x; x[4 * q + 1] = v.y; x[4 * q + 2] = v.z; x[4 * q + 3] = v.w;
    }
  }
}

// 16 f32 values of this thread's row as one 64-byte row of a 32 x 16 f32 box (the same
// 64-byte swizzle as a bf16 32-column row)
__device__ __forceinline__ void stage_half(uint8_t* slot, int lane, const float* x) {
  uint8_t* row = slot + lane * 64;
  const int sw = (lane >> 1) & 3;
#pragma unroll
  for (int q = 0; q < 4; ++q)
    *reinterpret_cast<float4*>(row + ((q ^ sw) << 4)) = make_float4(x[4 * q], x[4 * q + 1], x[4 * q + 2], x[4 * q + 3]);
}

// Stores one 32-row x 32-column chunk (rows row0.., columns col..) of this warp through the
// staging area and TMA tensor stores: bf16 as one 2 KB box, f32 as two 32 x 16 boxes of 2 KB.
// `slot_i` counts the warp's stores; two_slots: the area holds two 2 KB slots, used in turn,
// so a box is staged while the previous one is still being read.
__device__ __forceinline__ void store_chunk(const CUtensorMap* tm, uint8_t* staging, int& slot_i,
                                           int dt, int lane, const float* x, int col, int row0,
                                           bool two_slots) {
#pragma unroll
  for (int h = 0; h < (dt == DT_BF16 ? 1 : 2); ++h) {
    uint8_t* slot = staging + (two_slots ? (slot_i & 1) * (SLOT_BYTES / 2) : 0);
    if (lane == 0) {  // the store that last used this slot has read it
      if (two_slots) bulk_wait_read<1>();
      else bulk_wait_read<0>();
    }
    __syncwarp();
    if (dt == DT_BF16) stage_row(slot, dt, lane, x);
    else stage_half(slot, lane, x + 16 * h);
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    __syncwarp();
    if (lane == 0) {
      tma_store_2d(tm, (uint32_t)__cvta_generic_to_shared(slot), col + 16 * h, row0);
      bulk_commit();
    }
    ++slot_i;
  }
}

// ---- stream-K partials ---------------------------------------------------------------------
// This thread's row (TMEM lane) of tile rows 32 quad.., output chunk cidx (columns 32 cidx..):
// float4 q of the row at ((cidx * 8 + q) * 128 + row) * 4.  L2 only (st.cg / ld.cg): the
// slot is written and read within the launch, by different SMs.
__device__ __forceinline__ void sk_put(float* slot, int cidx, int row, const float* v) {
  float4* d = reinterpret_cast<float4*>(slot) + (size_t)cidx * 8 * BM + row;
#pragma unroll
  for (int q = 0; q < 8; ++q)
    __stcg(d + q * BM, make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]));
}
__device__ __forceinline__ void sk_add(const float* slot, int cidx, int row, float* v) {
  const float4* s = reinterpret_cast<const float4*>(slot) + (size_t)cidx * 8 * BM + row;
#pragma unroll
  for (int q = 0; q < 8; ++q) {
    const float4 x = __ldcg(s + q * BM);
    v[4 * q] += x.x; v[4 * q + 1] += x.y; v[4 * q + 2] += x.z; v[4 * q + 3] += x.w;
  }
}
__device__ __forceinline__ void flag_release(unsigned* f) {
  asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(f), "r"(1u) : "memory");
}
__device__ __forceinline__ unsigned flag_acquire(const unsigned* f) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(f) : "memory");
  return v;
}
// Bounded wait (global timer) for a published partial; false on expiry or abort.
__device__ __noinline__ bool sk_wait(const unsigned* f, volatile int* abort_flag, unsigned* err) {
  if (flag_acquire(f) != 0u) return true;
  const uint64_t t0 = global_ns();
  for (uint32_t it = 1;; ++it) {
    if (flag_acquire(f) != 0u) return true;
    if ((it & 63) == 0) {
      if (*abort_flag) return false;
      if (global_ns() - t0 > kWaitLimitNs) {
        *abort_flag = 1;
        set_dev_error(err, RA_DEVERR_TIMEOUT);
        return false;
      }
    }
  }
}

// Bias of one row's 32-column chunk [n, n + 32) (read from registers of the warp).
template <int EPI>
struct EpiIn {
  float bias[32];
};

// GELU of 8 values, kept out of line: the epilogue then carries one copy of its code instead
// of one per element, which keeps the hot loop inside the instruction cache.
struct F8 {
  float v[8];
};
__device__ __forceinline__ F8 gelu8(F8 x) {
#pragma unroll
  for (int i = 0; i < 8; i += 2) {
    const float2 y = gelu2(make_float2(x.v[i], x.v[i + 1]));
    x.v[i] = y.x;
    x.v[i + 1] = y.y;
  }
  return x;
}
// GELU(u) into x and GELU'(u) into d for 8 values, out of line for the same reason
struct F8x2 {
  F8 y, d;
};
__device__ __forceinline__ F8x2 gelu_both8(F8 x) {
  F8x2 r;
#pragma unroll
  for (int i = 0; i < 8; i += 2) {
    float2 y, d;
    gelu_both2(make_float2(x.v[i], x.v[i + 1]), y, d);
    r.y.v[i] = y.x; r.y.v[i + 1] = y.y;
    r.d.v[i] = d.x; r.d.v[i + 1] = d.y;
  }
  return r;
}

// One warp's 32 x 32 chunk of output C of the STORE and BIAS_GELU epilogues: rows row0..,
// columns n.. (this thread holds row row0 + lane in v).
template <int EPI>
__device__ __forceinline__ void epi_chunk(const TcParams& p, const CUtensorMap* tmC,
                                          const CUtensorMap* tmC2, uint8_t* staging, int& slot_i,
                                          int lane, int row0, int n, float* v, const EpiIn<EPI>& in,
                                          bool ts) {
#pragma unroll
  for (int i = 0; i < 32; i += 2) {
    const float2 y = __fadd2_rn(make_float2(v[i], v[i + 1]), make_float2(in.bias[i], in.bias[i + 1]));
    v[i] = y.x;
    v[i + 1] = y.y;
  }
  if (EPI == EPI_STORE) {
    store_chunk(tmC, staging, slot_i, p.c_dtype, lane, v, n, row0, ts);
  } else if (EPI == EPI_BIAS_GELU) {
    if (p.C) store_chunk(tmC, staging, slot_i, p.c_dtype, lane, v, n, row0, ts);
#pragma unroll
    for (int j = 0; j < 32; j += 8) {
      F8 x;
#pragma unroll
      for (int i = 0; i < 8; ++i) x.v[i] = v[j + i];
      x = gelu8(x);
#pragma unroll
      for (int i = 0; i < 8; ++i) v[j + i] = x.v[i];
    }
    store_chunk(tmC2, staging, slot_i, p.c2_dtype, lane, v, n, row0, ts);
  } else if (EPI == EPI_BIAS_GELU_G) {
    // GELU'(u) (bf16) goes into its staging slot 8 values at a time as they are computed, so
    // no second 32-value array stays live (this is what lets the epilogue run 12 warps);
    // GELU(u) replaces u in v and leaves through the usual chunk store
    uint8_t* slot = staging + (ts ? (slot_i & 1) * (SLOT_BYTES / 2) : 0);
    if (p.C) {
      if (lane == 0) {  // the store that last used this slot has read it
        if (ts) bulk_wait_read<1>();
        else bulk_wait_read<0>();
      }
      __syncwarp();
    }
    uint8_t* row = slot + lane * 64;
    const int sw = (lane >> 1) & 3;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      F8 x;
#pragma unroll
      for (int i = 0; i < 8; ++i) x.v[i] = v[8 * q + i];
      const F8x2 r = gelu_both8(x);
#pragma unroll
      for (int i = 0; i < 8; ++i) v[8 * q + i] = r.y.v[i];
      if (p.C) {
        uint4 u;
        u.x = pack_bf16x2(r.d.v[0], r.d.v[1]);
        u.y = pack_bf16x2(r.d.v[2], r.d.v[3]);
        u.z = pack_bf16x2(r.d.v[4], r.d.v[5]);
        u.w = pack_bf16x2(r.d.v[6], r.d.v[7]);
        *reinterpret_cast<uint4*>(row + ((q ^ sw) << 4)) = u;
      }
    }
    if (p.C) {
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      __syncwarp();
      if (lane == 0) {
        tma_store_2d(tmC, (uint32_t)__cvta_generic_to_shared(slot), n, row0);
        bulk_commit();
      }
      ++slot_i;
    }
    store_chunk(tmC2, staging, slot_i, p.c2_dtype, lane, v, n, row0, ts);
  }
}

// Tile order: groups of 8 M-tiles swept across N, so that CTAs running at the same time
// share A rows and B columns in L2.
__device__ __forceinline__ void tile_coords(int tile, int m_tiles, int n_tiles, int& mt, int& nt) {
  constexpr int GM = 8;
  const int per_group = GM * n_tiles;
  const int grp = tile / per_group, in = tile % per_group;
  const int gsz = min(GM, m_tiles - grp * GM);
  mt = grp * GM + in % gsz;
  nt = in / gsz;
}

// ---- the kernel -------------------------------------------------------------------------------
template <int BN, int EPI>
__global__ void __launch_bounds__(EpiTraits<EPI>::THREADS, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ CUtensorMap tmC, const __grid_constant__ CUtensorMap tmC2,
                   const __grid_constant__ CUtensorMap tmX, const TcParams p) {
  constexpr int EW = EpiTraits<EPI>::WARPS;
  using Cfg = TileCfg<BN, EpiTraits<EPI>::AUX, EW>;
  constexpr int STAGES = Cfg::STAGES;
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[STAGES], empty_bar[STAGES];
  __shared__ __align__(8) uint64_t tfull_bar[2], tempty_bar[2], drain_bar;
  __shared__ __align__(8) uint64_t aux_bar[EW][2];  // TMA loads of AUX operands
  __shared__ uint32_t tmem_base_sh;
  __shared__ volatile int abort_sh;

  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const uint32_t smem_base = smem_u32(smem);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull_bar[a], 1);
      mbar_init(&tempty_bar[a], EW);
    }
    mbar_init(&drain_bar, 1);
    for (int w = 0; w < EW; ++w) {
      mbar_init(&aux_bar[w][0], 1);
      mbar_init(&aux_bar[w][1], 1);
    }
    abort_sh = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 0 && lane == 0) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmA)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmB)) : "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(&tmem_base_sh)),
                 "r"((uint32_t)Cfg::TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = tmem_base_sh;
  // the set-up above overlaps the previous kernel's tail; operands are read only after it
  pdl_wait();
  pdl_trigger();
  Sched sch;
  sch.init(p, blockIdx.x, gridDim.x);

  if (warp == 0) {
    // ------------------------------------------------------------------ TMA producer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int pending_phase[STAGES];
      for (int s = 0; s < STAGES; ++s) pending_phase[s] = -1;
      bool ok = true;
      for (int u = 0; ok && u < sch.count(); ++u) {
        int tile, kb0, kb1, kind;
        sch.unit(u, tile, kb0, kb1, kind);
        int mt, nt;
        tile_coords(tile, p.m_tiles, p.n_tiles_n, mt, nt);
        const int m0 = mt * BM, n0 = nt * BN;
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(&empty_bar[stage], phase ^ 1u, &abort_sh, p.err)) { ok = false; break; }
          mbar_expect_tx(&full_bar[stage], Cfg::STAGE_BYTES);
          const uint32_t sa = smem_base + stage * Cfg::STAGE_BYTES;
          tma_load_2d(&tmA, sa, &full_bar[stage], kb * BK, m0);
          if (p.b_kn == 2) {
            tma_load_3d(&tmB, sa + Cfg::A_BYTES, &full_bar[stage], 0, kb * BK, n0 / 64);
          } else if (p.b_kn) {
            // rows kb*BK.. of B [K, N]: one 64-column swizzle atom (8 KB) per 64 columns
#pragma unroll
            for (int a = 0; a < BN / 64; ++a)
              tma_load_2d(&tmB, sa + Cfg::A_BYTES + a * 8192, &full_bar[stage], n0 + 64 * a, kb * BK);
          } else {
            tma_load_2d(&tmB, sa + Cfg::A_BYTES, &full_bar[stage], kb * BK, n0);
          }
          pending_phase[stage] = (int)phase;
          if (++stage == STAGES) { stage = 0; phase ^= 1u; }
        }
      }
      if (!ok) {  // let every copy this thread started land before the CTA goes away
        volatile int no_abort = 0;
        for (int s = 0; s < STAGES; ++s)
          if (pending_phase[s] >= 0) mbar_wait(&full_bar[s], (uint32_t)pending_phase[s], &no_abort, nullptr);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idesc = p.b_kn ? idesc_bf16_bmn(BM, BN) : idesc_bf16(BM, BN);
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool ok = true;
      for (int u = 0; ok && u < sch.count(); ++u) {
        int tile, kb0, kb1, kind;
        sch.unit(u, tile, kb0, kb1, kind);
        if (!mbar_wait(&tempty_bar[acc], acc_phase ^ 1u, &abort_sh, p.err)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * BN);
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(&full_bar[stage], phase, &abort_sh, p.err)) { ok = false; break; }
          tc_fence_after();
          const uint32_t sa = smem_base + stage * Cfg::STAGE_BYTES;
          const uint64_t adesc = sdesc_sw128(sa);
          // K-major B: advance 16 elements = 32 bytes inside the swizzle atom; [K, N] B
          // (MN-major): advance 16 rows = 2048 bytes, atoms along N 8 KB apart
          const uint64_t bdesc = p.b_kn ? sdesc_mn_sw128_lbo(sa + Cfg::A_BYTES, 8192) : sdesc_sw128(sa + Cfg::A_BYTES);
          const uint64_t bstep = p.b_kn ? 128u : 2u;
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)
            umma_bf16(d_tmem, adesc + (uint64_t)(2 * k), bdesc + bstep * (uint64_t)k, idesc,
                      (kb != kb0 || k != 0) ? 1u : 0u);
          umma_commit(&empty_bar[stage]);
          if (++stage == STAGES) { stage = 0; phase ^= 1u; }
        }
        if (!ok) break;
        umma_commit(&tfull_bar[acc]);
        if (++acc == 2) { acc = 0; acc_phase ^= 1u; }
      }
      // all MMAs issued by this thread complete before TMEM and shared memory are released
      umma_commit(&drain_bar);
      volatile int no_abort = 0;
      mbar_wait(&drain_bar, 0, &no_abort, nullptr);
    }
  } else {
    // ------------------------------------------------------------------ epilogue (warps 2..9)
    const int quad = warp & 3;             // TMEM lanes 32*quad .. 32*quad + 31
    const int half = (warp - 2) >> 2;      // which part of the tile's columns (EW / 4 parts)
    constexpr int PARTS = EW / 4;
    uint8_t* staging = smem + STAGES * Cfg::STAGE_BYTES + (warp - 2) * Cfg::WARP_STAGING;
    const bool two_slots = true;  // every output box is 2 KB
    int slot_i = 0;
    int acc = 0;
    uint32_t acc_phase = 0;
    int aux_i = 0;                         // AUX chunks issued by this warp (region = aux_i & 1)
    uint32_t aux_phase[2] = {0u, 0u};
    int aux_waited = 0;                    // AUX chunks whose load this warp has waited for
    uint64_t* abar = aux_bar[warp - 2];
    // AUX: TMA load of the operand chunk (rows row0.., output columns n..) into a region
    const int rbytes = (EPI == EPI_MUL && p.aux_dtype == DT_BF16) ? SLOT_BYTES / 2 : SLOT_BYTES;
    const int nreg = SLOT_BYTES / rbytes;
    auto aux_issue = [&](int row0_, int n_) {
      const int reg = aux_i % nreg;
      uint8_t* region = staging + reg * rbytes;
      if (lane == 0) {
        bulk_wait_read<0>();  // no tensor store still reads this region
        uint64_t* bar = &abar[reg];
        if (EPI == EPI_DSWIGLU) {
          const int gc = (n_ >> 6) * 128 + (n_ & 63);
          mbar_expect_tx(bar, 4096);
          tma_load_2d(&tmX, smem_u32(region), bar, gc, row0_);
          tma_load_2d(&tmX, smem_u32(region + 2048), bar, gc + 64, row0_);
        } else {
          mbar_expect_tx(bar, p.aux_dtype == DT_BF16 ? 2048 : 4096);
          tma_load_2d(&tmX, smem_u32(region), bar, n_, row0_);
        }
      }
      ++aux_i;
    };
    bool ok = true;
    const int ew = warp - 2;
    for (int u = 0; ok && u < sch.count(); ++u) {
      int tile, kb0, kb1, kind;
      sch.unit(u, tile, kb0, kb1, kind);
      int mt, nt;
      tile_coords(tile, p.m_tiles, p.n_tiles_n, mt, nt);
      const int m0 = mt * BM, n0 = nt * BN;
      const int row0 = m0 + quad * 32;
      const int cbeg = half * (BN / 2), cend = cbeg + BN / 2;
      // the first operand chunk is fetched while the main loop of this tile still runs
      if (EpiTraits<EPI>::AUX && n0 + cbeg < p.N && row0 < p.M) aux_issue(row0, n0 + cbeg);
      // bias of this warp's columns (BN / 2 floats, one 128-byte line per 32) brought into L1
      // while the accumulator is still being produced; the chunks then read it with
      // broadcast vector loads
      // (STORE / GELU: this warp's chunks are half, half + PARTS, ... of the tile's BN / 32)
      if ((EPI == EPI_STORE || EPI == EPI_BIAS_GELU || EPI == EPI_BIAS_GELU_G) && p.bias &&
          half + PARTS * lane < BN / 32 && n0 + 32 * (half + PARTS * lane) < p.N)
        asm volatile("prefetch.global.L1 [%0];" ::"l"(p.bias + n0 + 32 * (half + PARTS * lane)));
      if (!mbar_wait(&tfull_bar[acc], acc_phase, &abort_sh, p.err)) break;
      tc_fence_after();
      const uint32_t tbase = tmem_base + ((uint32_t)(quad * 32) << 16) + (uint32_t)(acc * BN);
      // finisher: the partials of CTAs src0 .. blockIdx.x - 1 (this warp's rows and columns)
      // must be published before they are added
      const int src0 = (EpiTraits<EPI>::SK && kind == 2) ? Sched::first_source(p, tile - p.dp_tiles) : 0;
      if (EpiTraits<EPI>::SK && kind == 2) {
        bool got = true;
        if (lane == 0)
          for (int cc = src0; got && cc < (int)blockIdx.x; ++cc)
            got = sk_wait(p.sk_flags + cc * SK_MAX_WARPS + ew, &abort_sh, p.err);
        if (!__shfl_sync(0xffffffffu, got ? 1 : 0, 0)) break;
      }
      if (EPI == EPI_SWIGLU) {
        // per 128-column block: gate columns [0, 64), up columns [64, 128); the two warps of
        // a quadrant split each block's 64 gate columns
#pragma unroll 1
        for (int blk = 0; blk < BN; blk += 128) {
          const int c0 = half * 32;
          float g[32], u[32];
          tmem_ld32(tbase + blk + c0, g);
          tmem_ld32(tbase + blk + 64 + c0, u);
          const int ng = n0 + blk + c0;           // packed gate column
          if (ng < p.N && row0 < p.M) {
            if (p.C) {
              store_chunk(&tmC, staging, slot_i, p.c_dtype, lane, g, ng, row0, two_slots);
              store_chunk(&tmC, staging, slot_i, p.c_dtype, lane, u, ng + 64, row0, two_slots);
            }
#pragma unroll
            for (int i = 0; i < 32; ++i) g[i] = silu_f(g[i]) * u[i];
            store_chunk(&tmC2, staging, slot_i, p.c2_dtype, lane, g, (n0 + blk) / 2 + c0, row0, two_slots);
          }
        }
      } else if (EpiTraits<EPI>::AUX) {
#pragma unroll 1
        for (int c0 = cbeg; c0 < cend; c0 += 32) {
          if (!(n0 + c0 < p.N && row0 < p.M)) break;  // live chunks form a prefix
          uint32_t r[32];
          tmem_ld32_issue(tbase + c0, r);
          const int reg = (aux_i - 1) % nreg;        // region of this chunk's operand
          uint8_t* region = staging + reg * rbytes;
          if (!mbar_wait(&abar[reg], aux_phase[reg], &abort_sh, p.err)) { ok = false; tmem_wait32(r); break; }
          aux_phase[reg] ^= 1u;
          ++aux_waited;
          float x1[32], x2[32];
          if (EPI == EPI_DSWIGLU) {
            unstage_row(region, DT_BF16, lane, x1);          // gate
            unstage_row(region + 2048, DT_BF16, lane, x2);   // up
          } else {
            unstage_row(region, p.aux_dtype, lane, x1);
          }
          __syncwarp();  // every lane has its operand row before the region is reused
          const bool more = c0 + 32 < cend && n0 + c0 + 32 < p.N;
          if (more && nreg == 2) aux_issue(row0, n0 + c0 + 32);
          tmem_wait32(r);
          float* v = reinterpret_cast<float*>(r);
          if (EPI == EPI_MUL) {
#pragma unroll
            for (int i = 0; i < 32; i += 2) {
              const float2 y = __fmul2_rn(make_float2(v[i], v[i + 1]), make_float2(x1[i], x1[i + 1]));
              v[i] = y.x;
              v[i + 1] = y.y;
            }
            store_chunk(&tmC, region, slot_i, p.c_dtype, lane, v, n0 + c0, row0, false);
          } else if (EPI == EPI_RESID) {
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] += x1[i];
            store_chunk(&tmC, region, slot_i, p.c_dtype, lane, v, n0 + c0, row0, false);
          } else {
            // d(h) -> d(gate), d(up) in the packed layout
            const int n = n0 + c0, gc = (n >> 6) * 128 + (n & 63);
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const float gt = x1[i], up = x2[i];
              x2[i] = v[i] * silu_f(gt);                 // d(up)
              v[i] = v[i] * up * silu_grad_f(gt);         // d(gate)
            }
            store_chunk(&tmC, region, slot_i, p.c_dtype, lane, v, gc, row0, false);
            store_chunk(&tmC, region + 2048, slot_i, p.c_dtype, lane, x2, gc + 64, row0, false);
          }
          if (more && nreg == 1) aux_issue(row0, n0 + c0 + 32);  // after the store has read it
        }
      } else {
        // STORE / BIAS_GELU: the TMEM load of chunk i + 1 is in flight while chunk i is
        // computed and stored; the accumulator is released as soon as its last chunk is in
        // registers, so the next tile's MMAs need not wait for these stores
        // this warp's chunks: tile columns 32 (half + PARTS i), i < nch
        const int nch = (BN / 32 - half + PARTS - 1) / PARTS;
        uint32_t ra[32], rb[32];
        auto col = [&](int i) { return 32 * (half + PARTS * i); };
        auto release = [&]() {
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&tempty_bar[acc]);
        };
        auto chunk = [&](int c0, uint32_t* r) {
          if (EpiTraits<EPI>::SK && kind == 1) {  // partial: the fp32 accumulator goes to this CTA's slot
            sk_put(p.sk_ws + (size_t)blockIdx.x * SK_SLOT_FLOATS, c0 / 32, quad * 32 + lane,
                   reinterpret_cast<const float*>(r));
            return;
          }
          // chunks entirely right of N or below M are skipped (warp-uniform); partial ones
          // are clipped by the tensor store
          if (n0 + c0 < p.N && row0 < p.M) {
            if (EpiTraits<EPI>::SK && kind == 2)
              for (int cc = src0; cc < (int)blockIdx.x; ++cc)
                sk_add(p.sk_ws + (size_t)cc * SK_SLOT_FLOATS, c0 / 32, quad * 32 + lane,
                       reinterpret_cast<float*>(r));
            EpiIn<EPI> in;
            // (N is a multiple of 8: a group of 8 that starts below N ends below it)
#pragma unroll
            for (int g8 = 0; g8 < 4; ++g8) {
              const int c = n0 + c0 + 8 * g8;
              float4 b0 = make_float4(0.f, 0.f, 0.f, 0.f), b1 = b0;
              if (p.bias && c < p.N) {
                b0 = __ldg(reinterpret_cast<const float4*>(p.bias + c));
                b1 = __ldg(reinterpret_cast<const float4*>(p.bias + c + 4));
              }
              float* bb = in.bias + 8 * g8;
              bb[0] = b0.x; bb[1] = b0.y; bb[2] = b0.z; bb[3] = b0.w;
              bb[4] = b1.x; bb[5] = b1.y; bb[6] = b1.z; bb[7] = b1.w;
            }
            epi_chunk<EPI>(p, &tmC, &tmC2, staging, slot_i, lane, row0, n0 + c0,
                           reinterpret_cast<float*>(r), in, two_slots);
          }
        };
        tmem_ld32_issue(tbase + col(0), ra);
#pragma unroll 1
        for (int i = 0; i < nch; i += 2) {
          tmem_wait32(ra);
          if (i + 1 < nch) tmem_ld32_issue(tbase + col(i + 1), rb);
          else release();
          chunk(col(i), ra);
          if (i + 1 < nch) {
            tmem_wait32(rb);
            if (i + 2 < nch) tmem_ld32_issue(tbase + col(i + 2), ra);
            else release();
            chunk(col(i + 1), rb);
          }
        }
      }
      if (EPI == EPI_STORE || EPI == EPI_BIAS_GELU || EPI == EPI_BIAS_GELU_G) {  // released above
        if (EpiTraits<EPI>::SK && kind == 1) {
          // publish this warp's part of the partial: every lane's stores are ordered before
          // the flag by the fence and the warp barrier, the flag store releases them
          __threadfence();
          __syncwarp();
          if (lane == 0) flag_release(p.sk_flags + blockIdx.x * SK_MAX_WARPS + ew);
        } else if (EpiTraits<EPI>::SK && kind == 2) {
          // the partials are consumed: clear their flags for the next launch (which reads
          // them only after this grid has completed)
          __syncwarp();
          if (lane == 0)
            for (int cc = src0; cc < (int)blockIdx.x; ++cc) p.sk_flags[cc * SK_MAX_WARPS + ew] = 0u;
        }
        if (++acc == 2) { acc = 0; acc_phase ^= 1u; }
        continue;
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty_bar[acc]);
      if (++acc == 2) { acc = 0; acc_phase ^= 1u; }
    }
    // an operand load issued but not consumed (only after an abort) lands before exit
    for (; aux_waited < aux_i; ++aux_waited) {
      const int reg = aux_waited % nreg;
      volatile int no_abort = 0;
      mbar_wait(&abar[reg], aux_phase[reg], &no_abort, nullptr);
      aux_phase[reg] ^= 1u;
    }
    if (lane == 0) bulk_wait_all();  // this warp's tensor stores are complete
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base),
                 "r"((uint32_t)Cfg::TMEM_COLS)
                 : "memory");
  }
}

// Failure-detection self-test: one thread waits, with the same bounded wait as the GEMM,
// on an mbarrier that nothing ever arrives on; the wait expires after limit_ns, records
// RA_DEVERR_TIMEOUT and the kernel returns normally.
__global__ void selftest_wait_kernel(unsigned* err, uint64_t limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ volatile int abort_sh;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort_sh = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  if (threadIdx.x == 0) mbar_wait(&bar, 0, &abort_sh, err, limit_ns);
}

// ---- host side --------------------------------------------------------------------------------
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static bool tried = false;
  if (!tried) {
    tried = true;
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

struct MapKey {
  const void* ptr;
  int64_t rows, cols, ld;
  int box_cols, box_rows, dtype, blocks;
  bool operator==(const MapKey& o) const {
    return ptr == o.ptr && rows == o.rows && cols == o.cols && ld == o.ld &&
           box_cols == o.box_cols && box_rows == o.box_rows && dtype == o.dtype && blocks == o.blocks;
  }
};
struct MapKeyHash {
  size_t operator()(const MapKey& k) const {
    size_t h = std::hash<const void*>()(k.ptr);
    h ^= std::hash<int64_t>()(k.rows * 1000003 + k.cols) + 0x9e3779b9 + (h << 6) + (h >> 2);
    h ^= std::hash<int64_t>()(k.ld * 31 + k.box_rows * 7 + k.box_cols * 131 + k.dtype + k.blocks * 1009) +
         0x9e3779b9 + (h << 6) + (h >> 2);
    return h;
  }
};

// Row-major [rows, cols] matrix with leading dimension ld (elements of dtype); box of
// box_cols x box_rows.  Operand loads (box 64 bf16 columns) use the 128-byte swizzle the
// MMA descriptors expect; output stores (32 bf16 or 16 f32 columns: 64-byte rows) and operand
// loads of the epilogues (32 columns) use the swizzle whose span is one box row, matching
// stage_row, stage_half and unstage_row.
// blocks > 0: the matrix (cols a multiple of box_cols) seen in 3-D as (box_cols columns, rows,
// cols / box_cols column blocks); one box of box_cols x box_rows x blocks then lands as
// `blocks` consecutive box_cols x box_rows tiles (the MN-major B operand atoms).
bool make_map(CUtensorMap* out, const void* ptr, int64_t rows, int64_t cols, int64_t ld,
              int box_cols, int box_rows, int dtype, int blocks = 0) {
  static std::mutex mu;
  static std::unordered_map<MapKey, CUtensorMap, MapKeyHash> cache;
  MapKey key{ptr, rows, cols, ld, box_cols, box_rows, dtype, blocks};
  std::lock_guard<std::mutex> lock(mu);
  auto it = cache.find(key);
  if (it != cache.end()) {
    *out = it->second;
    return true;
  }
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  const int es = dtype == DT_BF16 ? 2 : 4;
  const int row_bytes = box_cols * es;
  CUtensorMapSwizzle sw = row_bytes == 128 ? CU_TENSOR_MAP_SWIZZLE_128B
                        : row_bytes == 64  ? CU_TENSOR_MAP_SWIZZLE_64B
                                           : CU_TENSOR_MAP_SWIZZLE_NONE;
  const bool b3 = blocks > 0;
  if (b3 && cols % box_cols) return false;
  cuuint64_t gdim[3] = {(cuuint64_t)(b3 ? box_cols : cols), (cuuint64_t)rows, (cuuint64_t)(b3 ? cols / box_cols : 1)};
  cuuint64_t gstride[2] = {(cuuint64_t)ld * es, (cuuint64_t)box_cols * es};
  cuuint32_t box[3] = {(cuuint32_t)box_cols, (cuuint32_t)box_rows, (cuuint32_t)(b3 ? blocks : 1)};
  cuuint32_t estride[3] = {1, 1, 1};
  CUresult r = fn(out, dtype == DT_BF16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32,
                  b3 ? 3 : 2, const_cast<void*>(ptr), gdim, gstride, box, estride,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return false;
  if (cache.size() > 4096) cache.clear();
  cache.emplace(key, *out);
  return true;
}

template <int BN, int EPI>
cudaError_t launch(const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& c,
                   const CUtensorMap& c2, const CUtensorMap& x, const TcParams& p, int grid,
                   cudaStream_t st) {
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(gemm_tc_kernel<BN, EPI>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         TileCfg<BN, EpiTraits<EPI>::AUX, EpiTraits<EPI>::WARPS>::SMEM);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  const cudaError_t e = launch_pdl(gemm_tc_kernel<BN, EPI>, dim3(grid), dim3(EpiTraits<EPI>::THREADS),
                                   (size_t)TileCfg<BN, EpiTraits<EPI>::AUX, EpiTraits<EPI>::WARPS>::SMEM, st,
                                   a, b, c, c2, x, p);
  note_launch(1);
  return e != cudaSuccess ? e : cudaGetLastError();
}

template <int BN>
cudaError_t dispatch(const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& c,
                     const CUtensorMap& c2, const CUtensorMap& x, const TcParams& p, int grid,
                     cudaStream_t st) {
  switch (p.epi) {
    case EPI_STORE: return launch<BN, EPI_STORE>(a, b, c, c2, x, p, grid, st);
    case EPI_BIAS_GELU: return launch<BN, EPI_BIAS_GELU>(a, b, c, c2, x, p, grid, st);
    case EPI_MUL: return launch<BN, EPI_MUL>(a, b, c, c2, x, p, grid, st);
    case EPI_BIAS_GELU_G: return launch<BN, EPI_BIAS_GELU_G>(a, b, c, c2, x, p, grid, st);
    case EPI_RESID: return launch<BN, EPI_RESID>(a, b, c, c2, x, p, grid, st);
    case EPI_SWIGLU:
    case EPI_DSWIGLU:
      // the gate|up epilogues work on 128-column blocks: 128- and 256-wide tiles only
      if constexpr (BN % 128 == 0) {
        if (p.epi == EPI_SWIGLU) return launch<BN, EPI_SWIGLU>(a, b, c, c2, x, p, grid, st);
        return launch<BN, EPI_DSWIGLU>(a, b, c, c2, x, p, grid, st);
      }
      break;
  }
  return cudaErrorNotSupported;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

}  // namespace

bool tma_map_bf16(CUtensorMap* out, const void* ptr, int64_t rows, int64_t cols, int64_t ld, int box_cols,
                  int box_rows) {
  return make_map(out, ptr, rows, cols, ld, box_cols, box_rows, DT_BF16);
}

size_t gemm_sk_slot_bytes() { return (size_t)SK_SLOT_FLOATS * 4; }
int gemm_sk_flags_per_slot() { return SK_MAX_WARPS; }

cudaError_t selftest_wait(unsigned* err, uint64_t limit_ns, cudaStream_t st) {
  selftest_wait_kernel<<<1, 32, 0, st>>>(err, limit_ns);
  note_launch(1);
  return cudaGetLastError();
}

bool tc_available() {
  static int v = -1;
  if (v < 0) {
    int dev = 0, major = 0, minor = 0;
    v = 0;
    if (cudaGetDevice(&dev) == cudaSuccess &&
        cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) == cudaSuccess &&
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) == cudaSuccess)
      v = (major == 10 && minor == 3 && encode_fn() != nullptr) ? 1 : 0;
  }
  return v == 1;
}

cudaError_t gemm_tc(const GemmArgs& g, cudaStream_t st) {
  if (g.in_dtype != DT_BF16 || g.M <= 0 || g.N <= 0 || g.K <= 0) return cudaErrorNotSupported;
  // TMA: 16-byte aligned bases and row strides; epilogue: 8-column vector groups
  if (g.lda % 8 || g.ldb % 8 || g.K % 8 || g.N % 8 || !aligned16(g.A) || !aligned16(g.B))
    return cudaErrorNotSupported;
  const bool has_c = g.C != nullptr;
  if (has_c && (!aligned16(g.C) || g.ldc % 8)) return cudaErrorNotSupported;
  if (g.C2 && (!aligned16(g.C2) || g.ldc2 % 8)) return cudaErrorNotSupported;
  if (g.aux && (!aligned16(g.aux) || g.ldaux % 8)) return cudaErrorNotSupported;
  if (g.epi == EPI_SWIGLU && (g.N % 128 || !g.C2)) return cudaErrorNotSupported;
  // the GELU' output of EPI_BIAS_GELU_G is staged as bf16
  if (g.epi == EPI_BIAS_GELU_G && has_c && g.c_dtype != DT_BF16) return cudaErrorNotSupported;
  if (g.epi == EPI_DSWIGLU && g.N % 64) return cudaErrorNotSupported;
  if (!has_c && g.epi != EPI_BIAS_GELU && g.epi != EPI_BIAS_GELU_G && g.epi != EPI_SWIGLU)
    return cudaErrorNotSupported;

  const int sms = device_sm_count();
  const int m_tiles = (g.M + BM - 1) / BM;
  // tile width: fewest waves of 128 x BN tiles (time ~ waves x BN), weighting the narrower
  // tiles by their measured cost per column: a 128-wide tile carries more shared-memory
  // operand traffic per flop, and a 192-wide tile takes about as long as a 256-wide one
  // (measured: 0.96x the time of a 256-wide tile).  So 192 wins only where it saves a
  // whole wave at equal count, e.g. N = 768 at 4096 rows: 128 tiles in one wave instead of
  // 96 tiles of 256 columns on a third fewer SMs.
  auto cost = [&](int bn) {
    int tiles = m_tiles * ((g.N + bn - 1) / bn);
    int waves = (tiles + sms - 1) / sms;
    return (double)waves * bn * (bn == 128 ? 1.15 : bn == 192 ? 1.27 : 1.0);
  };
  int BNsel = (g.N <= 128 || cost(128) < cost(256)) ? 128 : 256;
  if (g.N > 128 && g.epi != EPI_SWIGLU && g.epi != EPI_DSWIGLU && cost(192) < cost(BNsel)) BNsel = 192;

  CUtensorMap ma, mb, mc, mc2, mx;
  memset(&mc, 0, sizeof mc);
  memset(&mc2, 0, sizeof mc2);
  memset(&mx, 0, sizeof mx);
  if (!make_map(&ma, g.A, g.M, g.K, g.lda, 64, BM, DT_BF16)) return cudaErrorNotSupported;
  // stored [K, N] B: one 3-D box per stage where N is a multiple of 64 (and the driver takes
  // the view), else BN / 64 boxes
  int b_kn = !g.b_kn ? 0 : g.N % 64 == 0 ? 2 : 1;
  if (b_kn == 2 && !make_map(&mb, g.B, g.K, g.N, g.ldb, 64, BK, DT_BF16, BNsel / 64)) b_kn = 1;
  if (b_kn == 1 && !make_map(&mb, g.B, g.K, g.N, g.ldb, 64, BK, DT_BF16)) return cudaErrorNotSupported;
  if (b_kn == 0 && !make_map(&mb, g.B, g.N, g.K, g.ldb, 64, BNsel, DT_BF16)) return cudaErrorNotSupported;
  // output maps: C is [M, N] except the packed d(gate|up) output of the SwiGLU' epilogue,
  // [M, 2N]; C2 is [M, N] (bias+GELU) or [M, N / 2] (h of the SwiGLU epilogue)
  if (has_c) {
    const int64_t cw = g.epi == EPI_DSWIGLU ? 2LL * g.N : g.N;
    // output boxes: 32 rows x 32 bf16 or x 16 f32 columns (64-byte rows)
    if (!make_map(&mc, g.C, g.M, cw, g.ldc, g.c_dtype == DT_BF16 ? 32 : 16, 32, g.c_dtype))
      return cudaErrorNotSupported;
  }
  if (g.C2) {
    const int64_t cw2 = g.epi == EPI_SWIGLU ? g.N / 2 : g.N;
    if (!make_map(&mc2, g.C2, g.M, cw2, g.ldc2, g.c2_dtype == DT_BF16 ? 32 : 16, 32, g.c2_dtype))
      return cudaErrorNotSupported;
  }
  // operand map of the GELU' / residual / SwiGLU' epilogues: [M, N], or the packed
  // [M, 2N] gate|up of SwiGLU' (always bf16)
  if (g.epi == EPI_MUL || g.epi == EPI_RESID || g.epi == EPI_DSWIGLU) {
    if (!g.aux) return cudaErrorNotSupported;
    if (g.epi == EPI_DSWIGLU && g.aux_dtype != DT_BF16) return cudaErrorNotSupported;
    const int64_t xw = g.epi == EPI_DSWIGLU ? 2LL * g.N : g.N;
    if (!make_map(&mx, g.aux, g.M, xw, g.ldaux, 32, 32, g.aux_dtype)) return cudaErrorNotSupported;
  }
  TcParams p;
  p.M = g.M; p.N = g.N; p.K = g.K;
  p.b_kn = b_kn;
  p.n_tiles_n = (g.N + BNsel - 1) / BNsel;
  p.m_tiles = m_tiles;
  p.num_tiles = m_tiles * p.n_tiles_n;
  p.k_blocks = (g.K + BK - 1) / BK;
  p.epi = g.epi;
  p.C = g.C; p.ldc = g.ldc; p.c_dtype = g.c_dtype;
  p.bias = g.bias;
  p.C2 = g.C2; p.ldc2 = g.ldc2; p.c2_dtype = g.c2_dtype;
  p.aux = g.aux; p.ldaux = g.ldaux; p.aux_dtype = g.aux_dtype;
  p.err = g.err;
  const int grid = p.num_tiles < sms ? p.num_tiles : sms;
  // Stream-K for the last, partial round of tiles (e.g. 256 tiles on 152 SMs: 104 tiles
  // would keep 104 SMs busy for a whole tile while 48 idle): their k-blocks are spread over
  // the CTAs.  Only after at least one full round (a single round stays one tile per CTA),
  // only where the round is not nearly full, only for the plain store epilogue, and only
  // where each CTA's share is at least 24 k-blocks: writing and reading back a tile's fp32
  // partials costs about as much as 8 to 12 k-blocks of MMA (measured on the BERT-large
  // shapes: 8192 x 1024 with K = 3072 or 4096 gain 3 to 4 us a launch, K = 1024 loses 4 us).
  p.dp_tiles = p.num_tiles;
  p.sk_ctas = 0;
  p.sk_iters = 0;
  p.sk_ws = g.sk_ws;
  p.sk_flags = g.sk_flags;
  const bool sk_epi = g.epi == EPI_STORE;
  if (sk_epi && g.sk_ws && g.sk_flags && grid <= g.sk_slots && p.num_tiles > grid) {
    const int rem = p.num_tiles % grid;
    const long long iters = (long long)rem * p.k_blocks;
    const int ctas = (int)std::min<long long>(grid, iters / 8);
    if (rem > 0 && rem * 100 < 85 * grid && ctas > rem && iters >= 24LL * ctas) {
      p.dp_tiles = p.num_tiles - rem;
      p.sk_ctas = ctas;
      p.sk_iters = (int)iters;
    }
  }
  return BNsel == 256 ? dispatch<256>(ma, mb, mc, mc2, mx, p, grid, st)
       : BNsel == 192 ? dispatch<192>(ma, mb, mc, mc2, mx, p, grid, st)
                      : dispatch<128>(ma, mb, mc, mc2, mx, p, grid, st);
}

}  // namespace ra
