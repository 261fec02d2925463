// k_attention_bwd_tc.cu -- attention backward on the 5th-generation tensor cores (tcgen05.mma
// with TMEM accumulators) for the encoder's short sequences: bf16, head_dim 64, no mask, no
// RoPE, S <= 256.  The softmax is recomputed from the saved row log-sum-exp (natural log of
// the scaled scores) and D = rowsum(dO * O) comes from the pre-pass:
//   P = exp(scale q k^T - lse),  dV = P^T dO,  dP = dO v^T,  dS = P * (dP - D),
//   dK = scale dS^T q,  dQ = scale dS k.
// Sequences are cut into 128-row blocks (NB = 1 or 2).  A CTA of 8 warps (two per TMEM lane
// quadrant, each taking 64 of a block's 128 columns) takes one block in one of two roles:
//   key pass for key block j (threads own key rows), over the query blocks i:
//     S^T = k_j q_i^T -> P^T (smem);  dV_j += P^T dO_i;  dP^T = v_j dO_i^T -> dS^T (smem, in
//     place of P^T once dV has read it);  dK_j += dS^T q_i
//   query pass for query block i (threads own query rows), over the key blocks j:
//     S = q_i k_j^T -> P (smem);  dP = dO_i v_j^T -> dS (smem, in place);  dQ_i += dS k_j
// so dQ, dK and dV each accumulate in TMEM over the other index in a fixed order
// (deterministic, no atomics).  P and dS are produced by the thread that owns their row, in
// the orientation the next product reads as its K-major A operand; the B operands of the
// three 64-wide products (dO_i, q_i, k_j) are read in place as MN-major blocks.  About 97 KB
// of shared memory and 256 TMEM columns per CTA: two CTAs share an SM.  Rows and columns at or beyond S are zero-filled and get
// P = 0.  Every wait on an MMA commit is bounded (global timer); on expiry the kernel records
// RA_DEVERR_TIMEOUT, lets its issued products finish, frees TMEM and returns.
#include "common.cuh"
#include "kernels.h"
#include "tcgen05.cuh"

namespace ra {
namespace {

using namespace tc;

constexpr float kLog2e = 1.4426950408889634f;
constexpr int BR = 128;          // rows of a query or key block
constexpr int HD = 64;           // head dim: one 128-byte swizzle atom of K
constexpr int NTHR = 256;        // 8 warps

__device__ __forceinline__ void cp_async16b(uint32_t dst, const void* src, bool valid) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(valid ? 16 : 0)
               : "memory");
}
// byte offset of 16-byte chunk j of row r in a 128-byte-row, 128-byte-swizzled tile
__device__ __forceinline__ uint32_t swz(int r, int j) { return (uint32_t)(r * 128 + ((j ^ (r & 7)) << 4)); }
__device__ __forceinline__ uint32_t pk2(float a, float b) {
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}
__device__ __forceinline__ float2 upk2(uint32_t u) {
  return __bfloat1622float2(*reinterpret_cast<__nv_bfloat162*>(&u));
}

// Shared memory (byte offsets; every tile 1024-byte aligned): four 128 x 64 blocks (128 rows
// of 128 bytes, K-major) -- the CTA's fixed block pair (k_j, v_j or q_i, dO_i) and the
// streamed pair -- and the staging block X (P^T / dS^T or P / dS: 128 x 128 as two atoms of
// [128][64]).  About 97 KB, so that two CTAs share an SM.
struct BwdPlan {
  static constexpr int T0 = 0, T1 = 16384, T2 = 32768, T3 = 49152, X = 65536, LSE = 98304,
                       DD = LSE + 512, BYTES = DD + 512;
  static constexpr uint32_t TMEM_COLS = 256;
  static constexpr uint32_t C_S = 0, C_A = 128, C_B = 192;  // S / dP; dV or dQ; dK
};

// cp.async copies of rows [r0, r0 + 128) of one head's 64 columns (base points at the head's
// first column of row 0; row stride ld elements) into a swizzled 128 x 64 tile; rows at or
// beyond S are zero-filled
__device__ __forceinline__ void load_block(uint32_t dst, const bf16* base, int ld, int r0, int S) {
  for (int e = threadIdx.x; e < BR * 8; e += NTHR) {
    const int r = e >> 3, j = e & 7, g = r0 + r;
    const bool ok = g < S;
    cp_async16b(dst + swz(r, j), base + (size_t)(ok ? g : 0) * ld + 8 * j, ok);
  }
}
// Descriptor of a 128 x 64 block read as an MN-major operand (the product's K runs along the
// block's rows, its N = 64 along the 128-byte rows: a single swizzle atom wide).  Eight-row
// K groups are 1024 bytes apart; the leading and stride byte offsets are both set to 1024,
// which is the K-group stride and leaves no second atom along N to address.
__device__ __forceinline__ uint64_t sdesc_mn_sw128(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)(1024 >> 4) << 16;
  d |= (uint64_t)(1024 >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}
// D[128 x N] (+)= A[128 x K] B^T, K = 64 (both K-major blocks, N = 128)
__device__ __forceinline__ void mma_qk(uint32_t d, uint32_t a, uint32_t b, uint32_t idesc) {
#pragma unroll
  for (int kk = 0; kk < HD / 16; ++kk)
    umma_bf16(d, sdesc_sw128(a + kk * 32), sdesc_sw128(b + kk * 32), idesc, kk > 0 ? 1u : 0u);
}
// D[128 x 64] (+)= X[128 x 128] B[128 x 64]: A = the staging block (K = 128 across its two
// atoms), B = a 128 x 64 block read MN-major (K = its rows, 16 rows = 2048 bytes per step)
__device__ __forceinline__ void mma_xb(uint32_t d, uint32_t x, uint32_t b, uint32_t idesc, bool acc) {
#pragma unroll
  for (int kk = 0; kk < BR / 16; ++kk)
    umma_bf16(d, sdesc_sw128(x + (kk >> 2) * (BR * 128) + (kk & 3) * 32), sdesc_mn_sw128(b + kk * 2048),
              idesc, (acc || kk > 0) ? 1u : 0u);
}

// blockIdx.x = (batch, head); blockIdx.y = role (0: key pass of key block blockIdx.z -> dK,
// dV; 1: query pass of query block blockIdx.z -> dQ)
template <int NB>
__global__ void __launch_bounds__(NTHR, 2) attn_bwd_tc_kernel(AttnArgs a) {
  using Pl = BwdPlan;
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
  const int H = a.n_heads * HD, ld = 3 * H, S = a.S;
  const bf16* qkv = reinterpret_cast<const bf16*>(a.qkv) + (size_t)b * S * ld + hh * HD;
  const bf16* dO = reinterpret_cast<const bf16*>(a.dO) + (size_t)b * S * H + hh * HD;
  bf16* dqkv = reinterpret_cast<bf16*>(a.dqkv) + (size_t)b * S * ld + hh * HD;
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
  // the key pass the thread's row is a key and the columns are queries; in the query pass
  // the row is a query.
  auto softmax_to_x = [&](int rbase, int cbase) {
#pragma unroll 1
    for (int h2 = 0; h2 < 2; ++h2) {
      float s[32];
      tmem_ld32(trow + Pl::C_S + c0 + 32 * h2, s);
#pragma unroll
      for (int g = 0; g < 4; ++g) {
        uint32_t w[4];
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          const int e = 8 * g + 2 * t, c = c0 + 32 * h2 + e;  // block column
          float p0, p1;
          if (keys) {  // row = key, column = query: lse per column
            const bool kr = rbase + row < S;
            p0 = (kr && cbase + c < S) ? exp2f(s[e] * sl2 - LSE[c]) : 0.f;
            p1 = (kr && cbase + c + 1 < S) ? exp2f(s[e + 1] * sl2 - LSE[c + 1]) : 0.f;
          } else {     // row = query, column = key: lse per row
            const bool qr = rbase + row < S;
            const float l = LSE[row];
            p0 = (qr && cbase + c < S) ? exp2f(s[e] * sl2 - l) : 0.f;
            p1 = (qr && cbase + c + 1 < S) ? exp2f(s[e + 1] * sl2 - l) : 0.f;
          }
          w[t] = pk2(p0, p1);
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
  // f * (TMEM columns [col, col + 64) of this thread's row): this half's 32 of them -> bf16
  // at dst (the row's 64 head columns) when the row is live.  Every lane of the warp runs
  // the TMEM load (a warp-wide instruction); only the store depends on the row.
  auto store_row = [&](uint32_t col, bf16* dst, float f, bool live) {
    float v[32];
    tmem_ld32(trow + col + 32 * half, v);
    if (!live) return;
#pragma unroll
    for (int g = 0; g < 4; ++g)
      *reinterpret_cast<uint4*>(dst + 32 * half + 8 * g) =
          make_uint4(pk2(v[8 * g] * f, v[8 * g + 1] * f), pk2(v[8 * g + 2] * f, v[8 * g + 3] * f),
                     pk2(v[8 * g + 4] * f, v[8 * g + 5] * f), pk2(v[8 * g + 6] * f, v[8 * g + 7] * f));
  };
  constexpr uint32_t ID128 = idesc_bf16(BR, BR);
  constexpr uint32_t ID64_MNB = idesc_bf16(BR, HD) | (1u << 16);  // B MN-major

  if (keys) {
    // ------------------------------------------------------------ key pass: dK_j, dV_j
    const int j = blk;
    load_block(sb + Pl::T0, qkv + H, ld, j * BR, S);       // k_j
    load_block(sb + Pl::T1, qkv + 2 * H, ld, j * BR, S);   // v_j
    for (int i = 0; i < NB && ok; ++i) {
      load_block(sb + Pl::T2, qkv, ld, i * BR, S);         // q_i
      load_block(sb + Pl::T3, dO, H, i * BR, S);           // dO_i
      load_stats(i * BR);
      copies_done();
      publish();
      if (tid == 0) {  // S^T = k_j q_i^T
        mma_qk(tmem + Pl::C_S, sb + Pl::T0, sb + Pl::T2, ID128);
        umma_commit(&bar);
      }
      pending = true;
      wait_mma();
      if (!ok) break;
      softmax_to_x(j * BR, i * BR);  // P^T
      publish();
      if (tid == 0) {  // dV_j += P^T dO_i; dP^T = v_j dO_i^T
        mma_xb(tmem + Pl::C_A, sb + Pl::X, sb + Pl::T3, ID64_MNB, i > 0);
        mma_qk(tmem + Pl::C_S, sb + Pl::T1, sb + Pl::T3, ID128);
        umma_commit(&bar);
      }
      pending = true;
      wait_mma();
      if (!ok) break;
      ds_in_x();  // dS^T over P^T (dV has read it)
      publish();
      if (tid == 0) {  // dK_j += dS^T q_i
        mma_xb(tmem + Pl::C_B, sb + Pl::X, sb + Pl::T2, ID64_MNB, i > 0);
        umma_commit(&bar);
      }
      pending = true;
      wait_mma();
    }
    if (ok) {
      const int kk = j * BR + row;
      bf16* dst = dqkv + (size_t)(kk < S ? kk : 0) * ld;
      store_row(Pl::C_A, dst + 2 * H, 1.f, kk < S);       // dV
      store_row(Pl::C_B, dst + H, a.scale, kk < S);       // dK
    }
  } else {
    // ------------------------------------------------------------ query pass: dQ_i
    const int i = blk;
    load_block(sb + Pl::T0, qkv, ld, i * BR, S);           // q_i
    load_block(sb + Pl::T1, dO, H, i * BR, S);             // dO_i
    load_stats(i * BR);
    for (int j = 0; j < NB && ok; ++j) {
      load_block(sb + Pl::T2, qkv + H, ld, j * BR, S);     // k_j
      load_block(sb + Pl::T3, qkv + 2 * H, ld, j * BR, S); // v_j
      copies_done();
      publish();
      if (tid == 0) {  // S = q_i k_j^T
        mma_qk(tmem + Pl::C_S, sb + Pl::T0, sb + Pl::T2, ID128);
        umma_commit(&bar);
      }
      pending = true;
      wait_mma();
      if (!ok) break;
      softmax_to_x(i * BR, j * BR);  // P (rows = queries)
      publish();  // S read before dP overwrites it
      if (tid == 0) {  // dP = dO_i v_j^T
        mma_qk(tmem + Pl::C_S, sb + Pl::T1, sb + Pl::T3, ID128);
        umma_commit(&bar);
      }
      pending = true;
      wait_mma();
      if (!ok) break;
      ds_in_x();  // dS over P
      publish();
      if (tid == 0) {  // dQ_i += dS k_j
        mma_xb(tmem + Pl::C_A, sb + Pl::X, sb + Pl::T2, ID64_MNB, j > 0);
        umma_commit(&bar);
      }
      pending = true;
      wait_mma();
    }
    if (ok) {
      const int q = i * BR + row;
      store_row(Pl::C_A, dqkv + (size_t)(q < S ? q : 0) * ld, a.scale, q < S);   // dQ
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

template <int NB>
cudaError_t launch_bwd_tc(const AttnArgs& a, cudaStream_t st) {
  auto k = attn_bwd_tc_kernel<NB>;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, BwdPlan::BYTES);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  cudaError_t e = launch_pdl(k, dim3(a.B * a.n_heads, 2, NB), dim3(NTHR), (size_t)BwdPlan::BYTES, st, a);
  note_launch(1);
  return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace

// expects D = rowsum(dO * O) in a.Dscratch and the forward's lse
cudaError_t attention_bwd_tc(const AttnArgs& a, cudaStream_t st) {
  if (!attention_tc_ok(a) || !a.lse || !a.Dscratch) return cudaErrorNotSupported;
  return a.S <= BR ? launch_bwd_tc<1>(a, st) : launch_bwd_tc<2>(a, st);
}

}  // namespace ra
