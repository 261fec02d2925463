// k_attention_tc.cu -- attention forward on the 5th-generation tensor cores (tcgen05.mma
// with TMEM accumulators) for the encoder's short sequences: bf16, head_dim 64, no mask, no
// RoPE, S <= 256.  CTA = 128 queries of one (batch, head), 8 warps (two per TMEM lane
// quadrant; each query row is shared by two threads, each taking half of the keys):
//   - one thread loads q (128 x 64), k and v (NK x 64; NK = S rounded up to 64) with three
//     TMA boxes into 128-byte-swizzled tiles, completion on an mbarrier;
//   - it issues S = q k^T (M 128, N NK, K 64) into TMEM columns [0, NK);
//   - each pair of threads reads its row of S from TMEM: row max, p = exp((s - max) * scale),
//     row sum (halves combined in a fixed order), and writes p (bf16) as the A operand of the
//     second product;
//   - O = p v (M 128, N 64, K NK) into TMEM columns [0, 64) (S is consumed by then), v read
//     as stored, MN-major through the descriptor (no transposed copy); O / sum and the
//     log-sum-exp (natural log of the scaled scores) go to memory.
// p reuses the shared memory of q and k, so two CTAs fit per SM.  All keys fit in one tile,
// so the softmax is exact in one pass (no running rescale).  Key rows at or beyond S hold
// the next sequence's keys (or, past the last token, the copy's zero fill): they get p = 0,
// and query rows beyond S are not stored.
#include "common.cuh"
#include "kernels.h"
#include "tcgen05.cuh"

namespace ra {
namespace {

using namespace tc;

constexpr float kLog2eT = 1.4426950408889634f;
constexpr int QT = 128;        // queries per CTA
constexpr int DH = 64;         // head dim (one 128-byte swizzle atom of K)

__device__ __forceinline__ uint32_t pack_bf16x2_tc(float a, float b) {
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}
// byte offset of 16-byte chunk j of row r in a 128-byte-row, 128-byte-swizzled tile
__device__ __forceinline__ uint32_t sw128(int r, int j) { return (uint32_t)(r * 128 + ((j ^ (r & 7)) << 4)); }

template <int NK>
struct AttnTcPlan {
  // v stays until O = p v; q and k are dead once S = q k^T is done, and p reuses them
  static constexpr int V_OFF = 0;                      // [NK][64] swizzled, MN-major B
  static constexpr int Q_OFF = NK * 128;               // [128][64] 16 KB
  static constexpr int K_OFF = Q_OFF + QT * 128;       // [NK][64]
  static constexpr int P_OFF = Q_OFF;                  // NK / 64 atoms of [128][64]
  static constexpr int BYTES = (K_OFF + NK * 128 > P_OFF + NK * 256) ? K_OFF + NK * 128 : P_OFF + NK * 256;
  static constexpr int SMEM = BYTES;                   // the extern array is 1024-byte aligned
  static constexpr uint32_t TMEM_COLS = NK;            // S; O reuses columns [0, 64)
};

__device__ __forceinline__ void tma_load_2d_at(const CUtensorMap* tm, uint32_t dst, uint64_t* bar, int c0, int c1) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tm)), "r"(c0), "r"(c1), "r"(smem_u32(bar))
      : "memory");
}

template <int NK>
__global__ void __launch_bounds__(256) attn_fwd_tc_kernel(const __grid_constant__ CUtensorMap tmQ,
                                                          const __grid_constant__ CUtensorMap tmKV, AttnArgs a) {
  using Pl = AttnTcPlan<NK>;
  constexpr int HALF = NK / 2;
  extern __shared__ __align__(1024) uint8_t smem[];
  __shared__ __align__(8) uint64_t mma_bar, load_bar;
  __shared__ uint32_t tmem_base_sh;
  __shared__ volatile int abort_sh;
  __shared__ float red[2][QT];  // per-row partials of the two halves
  const uint32_t sbase = smem_u32(smem);
  if (sbase & 1023u) {  // the swizzled operand tiles need 1024-byte alignment
    if (threadIdx.x == 0) set_dev_error(a.err, RA_DEVERR_BOUNDS);
    return;
  }
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int quad = warp & 3, half = warp >> 2;  // TMEM lane quadrant, column half
  const int bh = blockIdx.y, b = bh / a.n_heads, hh = bh % a.n_heads;
  const int H = a.n_heads * DH, S = a.S;
  const int q0 = blockIdx.x * QT;

  if (tid == 0) {
    mbar_init(&mma_bar, 1);
    mbar_init(&load_bar, 1);
    abort_sh = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmQ)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmKV)) : "memory");
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(&tmem_base_sh)), "r"(Pl::TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_sh;
  pdl_wait();
  pdl_trigger();

  // q, k and v: one box each from the [B S, 3 H] qkv matrix (x = the head's columns)
  if (tid == 0) {
    mbar_expect_tx(&load_bar, (uint32_t)(QT + 2 * NK) * 128);
    tma_load_2d_at(&tmQ, sbase + Pl::Q_OFF, &load_bar, hh * DH, b * S + q0);
    tma_load_2d_at(&tmKV, sbase + Pl::K_OFF, &load_bar, H + hh * DH, b * S);
    tma_load_2d_at(&tmKV, sbase + Pl::V_OFF, &load_bar, 2 * H + hh * DH, b * S);
  }
  bool ok = mbar_wait(&load_bar, 0, &abort_sh, a.err);
  tc_fence_after();

  // S = q k^T
  if (tid == 0 && ok) {
    constexpr uint32_t idesc = idesc_bf16(QT, NK);
    const uint64_t ad = sdesc_sw128(sbase + Pl::Q_OFF), bd = sdesc_sw128(sbase + Pl::K_OFF);
#pragma unroll
    for (int k = 0; k < DH / 16; ++k) umma_bf16(tmem, ad + (uint64_t)(2 * k), bd + (uint64_t)(2 * k), idesc, k > 0);
    umma_commit(&mma_bar);
  }
  if (ok) ok = mbar_wait(&mma_bar, 0, &abort_sh, a.err);
  tc_fence_before();
  __syncthreads();  // q and k are no longer read: p may overwrite them
  tc_fence_after();

  // softmax of row `row` over this thread's half of the keys
  const int row = 32 * quad + lane;
  const uint32_t trow = tmem + ((uint32_t)(32 * quad) << 16);
  const float sl2 = a.scale * kLog2eT;
  const int c0 = half * HALF;
  float mx = -INFINITY, sum = 0.f;
  // a chunk of 32 keys all below S (every chunk when S is a multiple of 32) skips the
  // per-key test: the softmax is issue-bound, so its instruction count sets its pace
  if (ok) {
#pragma unroll 1
    for (int c = c0; c < c0 + HALF; c += 32) {
      float s[32];
      tmem_ld32(trow + c, s);
      if (c + 32 <= S) {
#pragma unroll
        for (int i = 0; i < 32; ++i) mx = fmaxf(mx, s[i]);
      } else {
#pragma unroll
        for (int i = 0; i < 32; ++i)
          if (c + i < S) mx = fmaxf(mx, s[i]);
      }
    }
  }
  red[half][row] = mx;
  __syncthreads();
  mx = fmaxf(red[0][row], red[1][row]);
  // p = 2^(s sl2 - mx sl2): one fused multiply-add per key
  const float mxs = mx * sl2;
  if (ok) {
#pragma unroll 1
    for (int c = c0; c < c0 + HALF; c += 32) {
      float s[32];
      tmem_ld32(trow + c, s);
      const bool full = c + 32 <= S;
      uint8_t* atom = smem + Pl::P_OFF + (c >> 6) * (QT * 128);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        uint32_t w[4];
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          const int i = 8 * q + 2 * t;
          float p0 = ex2_fast(fmaf(s[i], sl2, -mxs)), p1 = ex2_fast(fmaf(s[i + 1], sl2, -mxs));
          if (!full) {
            p0 = c + i < S ? p0 : 0.f;
            p1 = c + i + 1 < S ? p1 : 0.f;
          }
          sum += p0 + p1;
          __nv_bfloat162 h2 = __floats2bfloat162_rn(p0, p1);
          w[t] = *reinterpret_cast<uint32_t*>(&h2);
        }
        *reinterpret_cast<uint4*>(atom + sw128(row, ((c & 63) >> 3) + q)) = make_uint4(w[0], w[1], w[2], w[3]);
      }
    }
  }
  __syncthreads();  // both halves have read their row maximum
  red[half][row] = sum;
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  sum = red[0][row] + red[1][row];

  // O = p v into TMEM columns [0, 64) (S is no longer read)
  if (tid == 0 && ok) {
    constexpr uint32_t idesc = idesc_bf16_bmn(QT, DH);
#pragma unroll
    for (int kk = 0; kk < NK / 16; ++kk) {
      const uint32_t pa = sbase + Pl::P_OFF + (kk >> 2) * (QT * 128) + (kk & 3) * 32;
      umma_bf16(tmem, sdesc_sw128(pa), sdesc_mn_sw128(sbase + Pl::V_OFF + kk * 2048), idesc, kk > 0);
    }
    umma_commit(&mma_bar);
  }
  if (ok) ok = mbar_wait(&mma_bar, 1, &abort_sh, a.err);
  tc_fence_after();
  if (ok) {
    const int q = q0 + row;
    const float inv = sum > 0.f ? 1.f / sum : 0.f;
    bf16* O = reinterpret_cast<bf16*>(a.O) + (size_t)(b * S + q) * H + hh * DH + 32 * half;
    float o[32];
    tmem_ld32(trow + 32 * half, o);
    if (q < S) {
#pragma unroll
      for (int g = 0; g < 4; ++g) {
        uint4 u;
        u.x = pack_bf16x2_tc(o[8 * g] * inv, o[8 * g + 1] * inv);
        u.y = pack_bf16x2_tc(o[8 * g + 2] * inv, o[8 * g + 3] * inv);
        u.z = pack_bf16x2_tc(o[8 * g + 4] * inv, o[8 * g + 5] * inv);
        u.w = pack_bf16x2_tc(o[8 * g + 6] * inv, o[8 * g + 7] * inv);
        *reinterpret_cast<uint4*>(O + 8 * g) = u;
      }
      if (a.lse && half == 0) a.lse[(size_t)bh * S + q] = mx * a.scale + logf(sum);
    }
  } else if (tid == 0) {
    // a wait gave up: the copies and any issued product finish before the shared memory and
    // TMEM are released (bounded waits)
    volatile int no_abort = 0;
    mbar_wait(&load_bar, 0, &no_abort, nullptr);
    mbar_wait(&mma_bar, 1, &no_abort, nullptr);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(Pl::TMEM_COLS)
                 : "memory");
  }
}

template <int NK>
cudaError_t launch_tc(const AttnArgs& a, cudaStream_t st) {
  auto k = attn_fwd_tc_kernel<NK>;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, AttnTcPlan<NK>::SMEM);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  // the qkv matrix [B S, 3 H]: q boxes of 64 columns x 128 rows, k and v boxes of NK rows
  const int H = a.n_heads * DH;
  CUtensorMap mq, mkv;
  if (!tma_map_bf16(&mq, a.qkv, (int64_t)a.B * a.S, 3LL * H, 3LL * H, DH, QT) ||
      !tma_map_bf16(&mkv, a.qkv, (int64_t)a.B * a.S, 3LL * H, 3LL * H, DH, NK))
    return cudaErrorNotSupported;
  cudaError_t e = launch_pdl(k, dim3((a.S + QT - 1) / QT, a.B * a.n_heads), dim3(256),
                             (size_t)AttnTcPlan<NK>::SMEM, st, mq, mkv, a);
  note_launch(1);
  return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace

bool attention_tc_ok(const AttnArgs& a) {
  // the TMA boxes start on 16-byte boundaries of the qkv rows
  return a.dtype == DT_BF16 && a.head_dim == DH && !a.causal && !a.rope && a.S >= 1 && a.S <= 256 &&
         (reinterpret_cast<uintptr_t>(a.qkv) & 15) == 0;
}

cudaError_t attention_fwd_tc(const AttnArgs& a, cudaStream_t st) {
  if (!attention_tc_ok(a)) return cudaErrorNotSupported;
  if (a.S <= 64) return launch_tc<64>(a, st);
  if (a.S <= 128) return launch_tc<128>(a, st);
  return launch_tc<256>(a, st);
}

}  // namespace ra
