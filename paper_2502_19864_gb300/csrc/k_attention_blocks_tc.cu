// k_attention_blocks_tc.cu -- attention over 128-row query and key blocks on the 5th-generation
// tensor cores (tcgen05.mma with TMEM accumulators): the backward for every bf16 shape of the
// step, and the forward of sequences longer than one key block (the decoder's).
//
// Backward: bf16, head_dim 64 or 128, optionally causal, with q and k either
// plain or carrying RoPE (rotated once in place by the forward, so the gradients of the
// rotated q and k get the rotation's transpose on the way out).  The softmax is recomputed
// from the saved row log-sum-exp (natural log of the scaled scores) and D = rowsum(dO * O)
// comes from the pre-pass:
//   P = exp(scale q k^T - lse),  dV = P^T dO,  dP = dO v^T,  dS = P * (dP - D),
//   dK = scale dS^T q,  dQ = scale dS k.
// Sequences are cut into 128-row blocks (NB = ceil(S / 128)).  A CTA of 8 warps (two per
// TMEM lane quadrant, each taking 64 of a block's 128 columns) takes one block in one of two
// roles:
//   key pass for key block j (threads own key rows), over the query blocks i (i >= j when
//   causal):
//     S^T = k_j q_i^T -> P^T (smem);  dV_j += P^T dO_i;  dP^T = v_j dO_i^T -> dS^T (smem, in
//     place of P^T once dV has read it);  dK_j += dS^T q_i
//   query pass for query block i (threads own query rows), over the key blocks j (j <= i
//   when causal):
//     S = q_i k_j^T -> P (smem);  dP = dO_i v_j^T -> dS (smem, in place);  dQ_i += dS k_j
// so dQ, dK and dV each accumulate in TMEM over the other index in a fixed order
// (deterministic, no atomics).  P and dS are produced by the thread that owns their row, in
// the orientation the next product reads as its K-major A operand; the B operands of the
// head-dim-wide products (dO_i, q_i, k_j) are read in place as MN-major blocks, one 64-wide
// swizzle atom (and one MMA) per 64 head dims.  Rows and columns at or beyond S, and keys
// after the query when causal, get P = 0.  Every wait on an MMA commit is bounded (global
// timer); on expiry the kernel records RA_DEVERR_TIMEOUT, lets its issued products finish,
// frees TMEM and returns.
#include "common.cuh"
#include "kernels.h"
#include "tcgen05.cuh"

namespace ra {
namespace {

using namespace tc;

constexpr float kLog2e = 1.4426950408889634f;
constexpr int BR = 128;          // rows of a query or key block
constexpr int NTHR = 256;        // 8 warps

__device__ __forceinline__ void cp_async16b(uint32_t dst, const void* src, bool valid) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(valid ? 16 : 0)
               : "memory");
}
__device__ __forceinline__ uint32_t pk2(float a, float b) {
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}
__device__ __forceinline__ float2 upk2(uint32_t u) {
  return __bfloat1622float2(*reinterpret_cast<__nv_bfloat162*>(&u));
}

// Shared memory (byte offsets; every tile 1024-byte aligned): four blocks of 128 rows x DH
// (DH / 64 swizzle atoms of [128][64], 16 KB each, K-major along the head dims) -- the CTA's
// fixed pair (k_j, v_j or q_i, dO_i) and the streamed pair -- and the staging block X (P^T /
// dS^T or P / dS: 128 x 128 as two atoms of [128][64]).  DH 64: about 97 KB and 256 TMEM
// columns (two CTAs per SM); DH 128: about 161 KB and 512 columns (one).
template <int DH>
struct BwdPlan {
  static constexpr int BLK = BR * DH * 2;
  static constexpr int T0 = 0, T1 = BLK, T2 = 2 * BLK, T3 = 3 * BLK, X = 4 * BLK, LSE = X + 32768,
                       DD = LSE + 512, BYTES = DD + 512;
  static constexpr uint32_t C_S = 0, C_A = 128, C_B = 128 + DH;  // S / dP; dV or dQ; dK
  static constexpr uint32_t TMEM_COLS = 128 + 2 * DH <= 256 ? 256 : 512;
};

// cp.async copies of rows [r0, r0 + 128) of one head's DH columns (base points at the head's
// first column of row 0; row stride ld elements) into a swizzled 128 x DH block; rows at or
// beyond S are zero-filled
template <int DH>
__device__ __forceinline__ void load_block(uint32_t dst, const bf16* base, int ld, int r0, int S) {
  constexpr int CH = DH / 8;  // 16-byte chunks per row
  for (int e = threadIdx.x; e < BR * CH; e += NTHR) {
    const int r = e / CH, j = e % CH, g = r0 + r;
    const bool ok = g < S;
    cp_async16b(dst + (j >> 3) * (BR * 128) + swz(r, j & 7), base + (size_t)(ok ? g : 0) * ld + 8 * j, ok);
  }
}
// D[128 x 128] = A B^T over K = DH (both K-major 128 x DH blocks)
template <int DH>
__device__ __forceinline__ void mma_qk(uint32_t d, uint32_t a, uint32_t b, uint32_t idesc) {
#pragma unroll
  for (int kk = 0; kk < DH / 16; ++kk) {
    const uint32_t o = (kk >> 2) * (BR * 128) + (kk & 3) * 32;
    umma_bf16(d, sdesc_sw128(a + o), sdesc_sw128(b + o), idesc, kk > 0 ? 1u : 0u);
  }
}
// D[128 x DH] (+)= X[128 x 128] B[128 x DH]: A = the staging block (K = 128 across its two
// atoms), B = a 128 x DH block read MN-major one 64-wide atom (and TMEM column range) at a
// time (K = its rows, 16 rows = 2048 bytes per step)
template <int DH>
__device__ __forceinline__ void mma_xb(uint32_t d, uint32_t x, uint32_t b, bool acc) {
  constexpr uint32_t idesc = idesc_bf16_bmn(BR, 64);
#pragma unroll
  for (int n = 0; n < DH / 64; ++n)
#pragma unroll
    for (int kk = 0; kk < BR / 16; ++kk)
      umma_bf16(d + 64 * n, sdesc_sw128(x + (kk >> 2) * (BR * 128) + (kk & 3) * 32),
                sdesc_mn_sw128(b + n * (BR * 128) + kk * 2048), idesc, (acc || kk > 0) ? 1u : 0u);
}

// blockIdx.x = (batch, head); blockIdx.y = role (0: key pass of key block blockIdx.z -> dK,
// dV; 1: query pass of query block blockIdx.z -> dQ)
template <int DH, bool CAUSAL, bool ROPE>
__global__ void __launch_bounds__(NTHR, DH == 64 ? 2 : 1) attn_bwd_tc_kernel(AttnArgs a) {
  using Pl = BwdPlan<DH>;
  extern __shared__ __align__(1024) uint8_t smem[];
  __shared__ __align__(8) uint64_t bar;
  __shared__ uint32_t tmem_sh;
  __shared__ volatile int abort_sh;
  const uint32_t sb = smem_u32(smem);
  if (sb & 1023u) {  // the swizzled operand tiles need 1024-byte alignment
    if (threadIdx.x == 0) set_dev_error(a.err, RA_DEVERR_BOUNDS);
    return;
  }
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int quad = warp & 3, half = warp >> 2;  // TMEM lane quadrant; 64-column half of a block
  const int bh = blockIdx.x, b = bh / a.n_heads, hh = bh % a.n_heads;
  const bool keys = blockIdx.y == 0;
  const int blk = blockIdx.z;                   // this CTA's key (or query) block
  const int S = a.S, NB = (S + BR - 1) / BR;
  const int H = a.n_heads * DH, ld = 3 * H;
  const bf16* qkv = reinterpret_cast<const bf16*>(a.qkv) + (size_t)b * S * ld + hh * DH;
  const bf16* dO = reinterpret_cast<const bf16*>(a.dO) + (size_t)b * S * H + hh * DH;
  bf16* dqkv = reinterpret_cast<bf16*>(a.dqkv) + (size_t)b * S * ld + hh * DH;
  const float* lse = a.lse + (size_t)bh * S;
  const float* Dv = a.Dscratch + (size_t)bh * S;
  float* LSE = reinterpret_cast<float*>(smem + Pl::LSE);
  float* DD = reinterpret_cast<float*>(smem + Pl::DD);
  const float sl2 = a.scale * kLog2e;

  if (tid == 0) {
    mbar_init(&bar, 1);
    abort_sh = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tmem_sh)),
                 "r"(Pl::TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  pdl_wait();
  pdl_trigger();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_sh;
  const uint32_t trow = tmem + ((uint32_t)(32 * quad) << 16);  // this warp's TMEM lanes
  const int row = 32 * quad + lane;                             // block row of this thread
  const int c0 = 64 * half;                                     // its 64 columns of a block
  uint8_t* xrow = smem + Pl::X + half * (BR * 128);             // its atom of the staging block
  uint32_t phase = 0;
  bool pending = false;  // a commit was issued and not yet waited for
  bool ok = true;

  // every thread waits for the last commit; then a uniform view of whether it arrived
  auto wait_mma = [&]() {
    if (ok) {
      mbar_wait(&bar, phase, &abort_sh, a.err);
      phase ^= 1u;
      pending = false;
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    ok = ok && abort_sh == 0;
  };
  // shared-memory writes by threads (and completed cp.async copies) -> visible to the
  // tensor cores; then a barrier
  auto publish = [&]() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
  };
  auto copies_done = [&]() {
    asm volatile("cp.async.commit_group;" ::: "memory");
    asm volatile("cp.async.wait_group 0;" ::: "memory");
  };
  auto load_stats = [&](int q0) {
    for (int r = tid; r < BR; r += NTHR) {
      const int q = q0 + r;
      LSE[r] = q < S ? lse[q] * kLog2e : 0.f;
      DD[r] = q < S ? Dv[q] : 0.f;
    }
  };
  // P (or P^T) of this thread's 64 columns from the scores in TMEM -> staging block X.  In
  // the key pass the thread's row is key rbase + row and the columns queries cbase + c; in
  // the query pass the row is a query and the columns keys.
  auto softmax_to_x = [&](int rbase, int cbase) {
    const int rg = rbase + row;
#pragma unroll 1
    for (int h2 = 0; h2 < 2; ++h2) {
      float s[32];
      tmem_ld32(trow + Pl::C_S + c0 + 32 * h2, s);
#pragma unroll
      for (int g = 0; g < 4; ++g) {
        uint32_t w[4];
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          float pp[2];
#pragma unroll
          for (int u = 0; u < 2; ++u) {
            const int e = 8 * g + 2 * t + u, c = c0 + 32 * h2 + e, cg = cbase + c;
            bool live = rg < S && cg < S;
            // causal: key <= query
            if (CAUSAL) live = live && (keys ? rg <= cg : cg <= rg);
            pp[u] = live ? ex2_fast(s[e] * sl2 - (keys ? LSE[c] : LSE[row])) : 0.f;
          }
          w[t] = pk2(pp[0], pp[1]);
        }
        *reinterpret_cast<uint4*>(xrow + swz(row, 4 * h2 + g)) = make_uint4(w[0], w[1], w[2], w[3]);
      }
    }
  };
  // dS = P (dP - D) over this thread's 64 columns, in place of P in X
  auto ds_in_x = [&]() {
#pragma unroll 1
    for (int h2 = 0; h2 < 2; ++h2) {
      float dp[32];
      tmem_ld32(trow + Pl::C_S + c0 + 32 * h2, dp);
#pragma unroll
      for (int g = 0; g < 4; ++g) {
        uint4* cell = reinterpret_cast<uint4*>(xrow + swz(row, 4 * h2 + g));
        const uint4 pv = *cell;
        const uint32_t pw[4] = {pv.x, pv.y, pv.z, pv.w};
        uint32_t w[4];
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          const int e = 8 * g + 2 * t, c = c0 + 32 * h2 + e;
          const float d0 = keys ? DD[c] : DD[row], d1 = keys ? DD[c + 1] : DD[row];
          const float2 p = upk2(pw[t]);
          w[t] = pk2(p.x * (dp[e] - d0), p.y * (dp[e + 1] - d1));
        }
        *cell = make_uint4(w[0], w[1], w[2], w[3]);
      }
    }
  };
  // f * (TMEM columns [col, col + DH) of this thread's row) -> bf16 at dst (the row's DH head
  // columns) when the row is live; this thread takes the head dims [16 DH/64 * half ...) in
  // rotate-half pairs (d, d + DH/2) so that the RoPE transpose has both members (rope: the
  // row's position s).  Every lane runs the TMEM loads (warp-wide); only the stores depend
  // on the row.
  auto store_row = [&](uint32_t col, bf16* dst, float f, bool live, bool rope, int s) {
    constexpr int HALFD = DH / 2, PER = HALFD / 2;  // pairs per thread: 16 (DH 64) or 32
    const int i0 = PER * half;
    float lo[32], hi[32];
    if (PER == 32) {
      tmem_ld32(trow + col + i0, lo);
      tmem_ld32(trow + col + HALFD + i0, hi);
    } else {  // DH 64: pairs (i, i + 32), i in [16 half, 16 half + 16)
      float t[32];
      tmem_ld32(trow + col, t);           // dims 0..31
      float u[32];
      tmem_ld32(trow + col + 32, u);      // dims 32..63
#pragma unroll
      for (int k = 0; k < 16; ++k) {  // compile-time indices on both sides (no local memory)
        lo[k] = half ? t[16 + k] : t[k];
        hi[k] = half ? u[16 + k] : u[k];
      }
    }
    if (!live) return;
#pragma unroll
    for (int k = 0; k < PER; ++k) {
      float x1 = lo[k] * f, x2 = hi[k] * f;
      if (rope) {
        float sn, cs;
        sincosf((float)s * rope_freq(i0 + k, DH, a.rope_theta), &sn, &cs);
        const float y1 = x1 * cs + x2 * sn, y2 = x2 * cs - x1 * sn;
        x1 = y1;
        x2 = y2;
      }
      lo[k] = x1;
      hi[k] = x2;
    }
#pragma unroll
    for (int g = 0; g < PER / 8; ++g) {
      *reinterpret_cast<uint4*>(dst + i0 + 8 * g) =
          make_uint4(pk2(lo[8 * g], lo[8 * g + 1]), pk2(lo[8 * g + 2], lo[8 * g + 3]),
                     pk2(lo[8 * g + 4], lo[8 * g + 5]), pk2(lo[8 * g + 6], lo[8 * g + 7]));
      *reinterpret_cast<uint4*>(dst + HALFD + i0 + 8 * g) =
          make_uint4(pk2(hi[8 * g], hi[8 * g + 1]), pk2(hi[8 * g + 2], hi[8 * g + 3]),
                     pk2(hi[8 * g + 4], hi[8 * g + 5]), pk2(hi[8 * g + 6], hi[8 * g + 7]));
    }
  };
  constexpr uint32_t ID128 = idesc_bf16(BR, BR);

  if (keys) {
    // ------------------------------------------------------------ key pass: dK_j, dV_j
    const int j = blk;
    load_block<DH>(sb + Pl::T0, qkv + H, ld, j * BR, S);       // k_j
    load_block<DH>(sb + Pl::T1, qkv + 2 * H, ld, j * BR, S);   // v_j
    const int i_first = CAUSAL ? j : 0;
    for (int i = i_first; i < NB && ok; ++i) {
      load_block<DH>(sb + Pl::T2, qkv, ld, i * BR, S);         // q_i
      load_block<DH>(sb + Pl::T3, dO, H, i * BR, S);           // dO_i
      load_stats(i * BR);
      copies_done();
      publish();
      if (tid == 0) {  // S^T = k_j q_i^T
        mma_qk<DH>(tmem + Pl::C_S, sb + Pl::T0, sb + Pl::T2, ID128);
        umma_commit(&bar);
      }
      pending = true;
      wait_mma();
      if (!ok) break;
      softmax_to_x(j * BR, i * BR);  // P^T
      publish();
      if (tid == 0) {  // dV_j += P^T dO_i; dP^T = v_j dO_i^T
        mma_xb<DH>(tmem + Pl::C_A, sb + Pl::X, sb + Pl::T3, i > i_first);
        mma_qk<DH>(tmem + Pl::C_S, sb + Pl::T1, sb + Pl::T3, ID128);
        umma_commit(&bar);
      }
      pending = true;
      wait_mma();
      if (!ok) break;
      ds_in_x();  // dS^T over P^T (dV has read it)
      publish();
      if (tid == 0) {  // dK_j += dS^T q_i
        mma_xb<DH>(tmem + Pl::C_B, sb + Pl::X, sb + Pl::T2, i > i_first);
        umma_commit(&bar);
      }
      pending = true;
      wait_mma();
    }
    if (ok) {
      const int kk = j * BR + row;
      bf16* dst = dqkv + (size_t)(kk < S ? kk : 0) * ld;
      store_row(Pl::C_A, dst + 2 * H, 1.f, kk < S, false, kk);      // dV
      store_row(Pl::C_B, dst + H, a.scale, kk < S, ROPE, kk);       // dK
    }
  } else {
    // ------------------------------------------------------------ query pass: dQ_i
    const int i = blk;
    load_block<DH>(sb + Pl::T0, qkv, ld, i * BR, S);           // q_i
    load_block<DH>(sb + Pl::T1, dO, H, i * BR, S);             // dO_i
    load_stats(i * BR);
    const int j_end = CAUSAL ? i + 1 : NB;
    for (int j = 0; j < j_end && ok; ++j) {
      load_block<DH>(sb + Pl::T2, qkv + H, ld, j * BR, S);     // k_j
      load_block<DH>(sb + Pl::T3, qkv + 2 * H, ld, j * BR, S); // v_j
      copies_done();
      publish();
      if (tid == 0) {  // S = q_i k_j^T
        mma_qk<DH>(tmem + Pl::C_S, sb + Pl::T0, sb + Pl::T2, ID128);
        umma_commit(&bar);
      }
      pending = true;
      wait_mma();
      if (!ok) break;
      softmax_to_x(i * BR, j * BR);  // P (rows = queries)
      publish();  // S read before dP overwrites it
      if (tid == 0) {  // dP = dO_i v_j^T
        mma_qk<DH>(tmem + Pl::C_S, sb + Pl::T1, sb + Pl::T3, ID128);
        umma_commit(&bar);
      }
      pending = true;
      wait_mma();
      if (!ok) break;
      ds_in_x();  // dS over P
      publish();
      if (tid == 0) {  // dQ_i += dS k_j
        mma_xb<DH>(tmem + Pl::C_A, sb + Pl::X, sb + Pl::T2, j > 0);
        umma_commit(&bar);
      }
      pending = true;
      wait_mma();
    }
    if (ok) {
      const int q = i * BR + row;
      store_row(Pl::C_A, dqkv + (size_t)(q < S ? q : 0) * ld, a.scale, q < S, ROPE, q);   // dQ
    }
  }

  if (pending) {
    // a wait gave up: let the issued products finish before TMEM is released
    volatile int no_abort = 0;
    mbar_wait(&bar, phase, &no_abort, nullptr);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(Pl::TMEM_COLS)
                 : "memory");
  }
}

template <int DH, bool CAUSAL, bool ROPE>
cudaError_t launch_bwd_tc(const AttnArgs& a, cudaStream_t st) {
  auto k = attn_bwd_tc_kernel<DH, CAUSAL, ROPE>;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, BwdPlan<DH>::BYTES);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  const int nb = (a.S + BR - 1) / BR;
  cudaError_t e = launch_pdl(k, dim3(a.B * a.n_heads, 2, nb), dim3(NTHR), (size_t)BwdPlan<DH>::BYTES, st, a);
  note_launch(1);
  return e != cudaSuccess ? e : cudaGetLastError();
}

// ---------------------------------------------------------------------------------------
// Forward over key blocks, two exact passes (no running rescale of the output):
//   pass 1: S = q_i k_j^T for every key block -> each thread's running max and sum of
//           exp over its 64 columns -> the row's log-sum-exp (halves combined in a fixed
//           order);
//   pass 2: S again -> P = exp(scale S - lse) (bf16, smem) -> O += P v_j (TMEM).
// The scores are computed twice (1.5x the forward flops) so that O accumulates exactly in
// TMEM and leaves it once.  CTA = 128 queries of one (batch, head), 8 warps (two per TMEM
// lane quadrant, each taking 64 of a key block's 128 columns).  Keys after the query (causal)
// or at or beyond S get P = 0; the output and lse of query rows at or beyond S are not
// written.  q and k arrive as the attention reads them (rotated in place for RoPE).
// Shared memory: q_i, k_j and v_j blocks (128 x DH each) and P (128 x 128, 32 KB).  At DH 128
// P takes k_j's space (exactly one block) once S has been computed; k_j is reloaded for the
// next key block after O += P v_j has read P.  That keeps a CTA at 98 KB: two CTAs per SM
// (256 TMEM columns each).  At DH 64 P has its own 32 KB after the blocks (80 KB).
template <int DH>
struct FwdPlan {
  static constexpr int BLK = BR * DH * 2;
  static constexpr int Q = 0, K = BLK, V = 2 * BLK, X = DH == 128 ? BLK : 3 * BLK;
  static constexpr int RED = DH == 128 ? 3 * BLK : 3 * BLK + 32768, BYTES = RED + 2048;
  static constexpr uint32_t C_S = 0, C_O = 128;
  static constexpr uint32_t TMEM_COLS = 128 + DH <= 256 ? 256 : 512;
};

// blockIdx.x counts query blocks from the last: with a causal mask the blocks with the most
// key blocks start first
template <int DH, bool CAUSAL>
__global__ void __launch_bounds__(NTHR, 2) attn_fwd_blocks_tc_kernel(AttnArgs a) {
  using Pl = FwdPlan<DH>;
  extern __shared__ __align__(1024) uint8_t smem[];
  __shared__ __align__(8) uint64_t bar;
  __shared__ uint32_t tmem_sh;
  __shared__ volatile int abort_sh;
  const uint32_t sb = smem_u32(smem);
  if (sb & 1023u) {  // the swizzled operand tiles need 1024-byte alignment
    if (threadIdx.x == 0) set_dev_error(a.err, RA_DEVERR_BOUNDS);
    return;
  }
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int quad = warp & 3, half = warp >> 2;
  const int S = a.S, NB = (S + BR - 1) / BR;
  const int i = NB - 1 - (int)blockIdx.x, bh = blockIdx.y, b = bh / a.n_heads, hh = bh % a.n_heads;
  const int H = a.n_heads * DH, ld = 3 * H;
  const bf16* qkv = reinterpret_cast<const bf16*>(a.qkv) + (size_t)b * S * ld + hh * DH;
  float (*red)[2][BR] = reinterpret_cast<float (*)[2][BR]>(smem + Pl::RED);  // [m | l][half][row]
  const float sl2 = a.scale * kLog2e;

  if (tid == 0) {
    mbar_init(&bar, 1);
    abort_sh = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tmem_sh)),
                 "r"(Pl::TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  pdl_wait();
  pdl_trigger();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_sh;
  const uint32_t trow = tmem + ((uint32_t)(32 * quad) << 16);
  const int row = 32 * quad + lane, q = i * BR + row;
  const int c0 = 64 * half;
  uint8_t* xrow = smem + Pl::X + half * (BR * 128);
  uint32_t phase = 0;
  bool pending = false;
  bool ok = true;
  auto wait_mma = [&]() {
    if (ok) {
      mbar_wait(&bar, phase, &abort_sh, a.err);
      phase ^= 1u;
      pending = false;
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    ok = ok && abort_sh == 0;
  };
  auto publish = [&]() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
  };
  auto copies_done = [&]() {
    asm volatile("cp.async.commit_group;" ::: "memory");
    asm volatile("cp.async.wait_group 0;" ::: "memory");
  };
  auto live = [&](int key) { return q < S && key < S && (!CAUSAL || key <= q); };
  constexpr uint32_t ID128 = idesc_bf16(BR, BR);
  const int j_end = CAUSAL ? i + 1 : NB;

  load_block<DH>(sb + Pl::Q, qkv, ld, i * BR, S);
  // ---- pass 1: the row's max and sum of exp (log2 units of the scaled scores)
  float m = -INFINITY, l = 0.f;
  for (int j = 0; j < j_end && ok; ++j) {
    load_block<DH>(sb + Pl::K, qkv + H, ld, j * BR, S);
    copies_done();
    publish();
    if (tid == 0) {
      mma_qk<DH>(tmem + Pl::C_S, sb + Pl::Q, sb + Pl::K, ID128);
      umma_commit(&bar);
    }
    pending = true;
    wait_mma();
    if (!ok) break;
#pragma unroll 1
    for (int h2 = 0; h2 < 2; ++h2) {
      float s[32];
      tmem_ld32(trow + Pl::C_S + c0 + 32 * h2, s);
      const int k0 = j * BR + c0 + 32 * h2;
      // a chunk whose 32 keys are all live for this row skips the per-key test
      const bool all_live = live(k0) && live(k0 + 31);
      float bm = -INFINITY;
      if (all_live) {
#pragma unroll
        for (int e = 0; e < 32; ++e) bm = fmaxf(bm, s[e] * sl2);
      } else {
#pragma unroll
        for (int e = 0; e < 32; ++e)
          if (live(k0 + e)) bm = fmaxf(bm, s[e] * sl2);
      }
      if (bm > m) {
        l *= exp2f(m - bm);
        m = bm;
      }
      if (all_live) {
#pragma unroll
        for (int e = 0; e < 32; ++e) l += ex2_fast(s[e] * sl2 - m);
      } else if (m > -INFINITY) {
#pragma unroll
        for (int e = 0; e < 32; ++e)
          if (live(k0 + e)) l += ex2_fast(s[e] * sl2 - m);
      }
    }
  }
  red[0][half][row] = m;
  red[1][half][row] = l;
  __syncthreads();
  const float m0 = red[0][0][row], m1 = red[0][1][row];
  const float M = fmaxf(m0, m1);
  const float L = M > -INFINITY ? red[1][0][row] * exp2f(m0 - M) + red[1][1][row] * exp2f(m1 - M) : 0.f;
  const float lse2 = M > -INFINITY ? M + log2f(L) : 0.f;
  // ---- pass 2: P = exp(scale S - lse), O += P v_j
  for (int j = 0; j < j_end && ok; ++j) {
    load_block<DH>(sb + Pl::K, qkv + H, ld, j * BR, S);
    asm volatile("cp.async.commit_group;" ::: "memory");
    load_block<DH>(sb + Pl::V, qkv + 2 * H, ld, j * BR, S);  // lands while S is computed
    asm volatile("cp.async.commit_group;" ::: "memory");
    asm volatile("cp.async.wait_group 1;" ::: "memory");      // k_j
    publish();
    if (tid == 0) {
      mma_qk<DH>(tmem + Pl::C_S, sb + Pl::Q, sb + Pl::K, ID128);
      umma_commit(&bar);
    }
    pending = true;
    wait_mma();  // k_j is free from here: P goes into its space
    if (!ok) break;
#pragma unroll 1
    for (int h2 = 0; h2 < 2; ++h2) {
      float s[32];
      tmem_ld32(trow + Pl::C_S + c0 + 32 * h2, s);
      const int k0 = j * BR + c0 + 32 * h2;
      const bool all_live = live(k0) && live(k0 + 31);
#pragma unroll
      for (int g = 0; g < 4; ++g) {
        uint32_t w[4];
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          const int e = 8 * g + 2 * t;
          float p0 = ex2_fast(s[e] * sl2 - lse2), p1 = ex2_fast(s[e + 1] * sl2 - lse2);
          if (!all_live) {
            p0 = live(k0 + e) ? p0 : 0.f;
            p1 = live(k0 + e + 1) ? p1 : 0.f;
          }
          w[t] = pk2(p0, p1);
        }
        *reinterpret_cast<uint4*>(xrow + swz(row, 4 * h2 + g)) = make_uint4(w[0], w[1], w[2], w[3]);
      }
    }
    asm volatile("cp.async.wait_group 0;" ::: "memory");  // v_j
    publish();
    if (tid == 0) {
      mma_xb<DH>(tmem + Pl::C_O, sb + Pl::X, sb + Pl::V, j > 0);
      umma_commit(&bar);
    }
    pending = true;
    wait_mma();
  }
  if (ok) {
    // O (already normalised) -> bf16; this thread takes head dims [DH/2 * half, + DH/2)
    bf16* O = reinterpret_cast<bf16*>(a.O) + ((size_t)b * S + (q < S ? q : 0)) * H + hh * DH + (DH / 2) * half;
#pragma unroll 1
    for (int c = 0; c < DH / 2; c += 32) {
      float o[32];
      tmem_ld32(trow + Pl::C_O + (DH / 2) * half + c, o);
      if (q < S) {
#pragma unroll
        for (int g = 0; g < 4; ++g)
          *reinterpret_cast<uint4*>(O + c + 8 * g) =
              make_uint4(pk2(o[8 * g], o[8 * g + 1]), pk2(o[8 * g + 2], o[8 * g + 3]),
                         pk2(o[8 * g + 4], o[8 * g + 5]), pk2(o[8 * g + 6], o[8 * g + 7]));
      }
    }
    if (a.lse && half == 0 && q < S) a.lse[(size_t)bh * S + q] = lse2 * 0.69314718055994531f;
  }
  if (pending) {
    volatile int no_abort = 0;
    mbar_wait(&bar, phase, &no_abort, nullptr);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(Pl::TMEM_COLS)
                 : "memory");
  }
}

template <int DH, bool CAUSAL>
cudaError_t launch_fwd_blocks(const AttnArgs& a, cudaStream_t st) {
  auto k = attn_fwd_blocks_tc_kernel<DH, CAUSAL>;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, FwdPlan<DH>::BYTES);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  const int nb = (a.S + BR - 1) / BR;
  cudaError_t e = launch_pdl(k, dim3(nb, a.B * a.n_heads), dim3(NTHR), (size_t)FwdPlan<DH>::BYTES, st, a);  // x: reversed
  note_launch(1);
  return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace

bool attention_fwd_blocks_tc_ok(const AttnArgs& a) {
  return a.dtype == DT_BF16 && (a.head_dim == 64 || a.head_dim == 128) && a.S >= 1 &&
         (!a.rope || a.qk_rotated);
}

cudaError_t attention_fwd_blocks_tc(const AttnArgs& a, cudaStream_t st) {
  if (!attention_fwd_blocks_tc_ok(a)) return cudaErrorNotSupported;
  if (a.head_dim == 64) return a.causal ? launch_fwd_blocks<64, true>(a, st) : launch_fwd_blocks<64, false>(a, st);
  return a.causal ? launch_fwd_blocks<128, true>(a, st) : launch_fwd_blocks<128, false>(a, st);
}

bool attention_bwd_tc_ok(const AttnArgs& a) {
  return a.dtype == DT_BF16 && (a.head_dim == 64 || a.head_dim == 128) && a.S >= 1 &&
         (!a.rope || a.qk_rotated) && a.lse && a.Dscratch;
}

// expects D = rowsum(dO * O) in a.Dscratch and the forward's lse
cudaError_t attention_bwd_tc(const AttnArgs& a, cudaStream_t st) {
  if (!attention_bwd_tc_ok(a)) return cudaErrorNotSupported;
  const bool rope = a.rope;  // q and k were rotated in place by the forward
  if (a.head_dim == 64) {
    if (a.causal) return rope ? launch_bwd_tc<64, true, true>(a, st) : launch_bwd_tc<64, true, false>(a, st);
    return rope ? launch_bwd_tc<64, false, true>(a, st) : launch_bwd_tc<64, false, false>(a, st);
  }
  if (a.causal) return rope ? launch_bwd_tc<128, true, true>(a, st) : launch_bwd_tc<128, true, false>(a, st);
  return rope ? launch_bwd_tc<128, false, true>(a, st) : launch_bwd_tc<128, false, false>(a, st);
}

}  // namespace ra
