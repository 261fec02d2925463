// k_attention_mma.cu -- fused attention forward and backward on the tensor cores
// (mma.sync m16n8k16, bf16 operands, fp32 accumulation) for the bf16 models.
//
// Per (batch, head): softmax(q k^T * scale [+ causal mask]) v with the online softmax, so
// the S x S scores never reach memory; the forward keeps only O and the row log-sum-exp.
// The backward recomputes P from q, k and that statistic: a dK/dV kernel holds 64 keys
// and streams the queries, a dQ kernel holds 64 queries and streams the keys (no atomics,
// deterministic).  RoPE (rotate-half) is applied to q and k as they enter shared memory and
// its transpose to dq and dk in registers before they are stored, so the saved q|k|v are
// the raw projections.  Warps own 16 rows; P and dS are fed back into the next product
// straight from the accumulator registers.
#include "common.cuh"
#include "kernels.h"

namespace ra {
namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

__device__ __forceinline__ void mma16816(float* d, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
      "{%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void ldsm4(uint32_t* r, const bf16* p) {
  uint32_t a = (uint32_t)__cvta_generic_to_shared(p);
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(a));
}
__device__ __forceinline__ void ldsm4t(uint32_t* r, const bf16* p) {
  uint32_t a = (uint32_t)__cvta_generic_to_shared(p);
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(a));
}
__device__ __forceinline__ uint32_t pk(float a, float b) {
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}

// A fragment of rows [r0, r0+16) x cols [c0, c0+16) of a row-major smem tile
__device__ __forceinline__ void frag_a(uint32_t* a, const bf16* s, int ld, int r0, int c0, int lane) {
  ldsm4(a, s + (size_t)(r0 + (lane & 7) + ((lane >> 3) & 1) * 8) * ld + c0 + (lane >> 4) * 8);
}
// B fragments of two n8 tiles where the smem tile is [n][k] (k contiguous): n rows
// [n0, n0+16), k cols [k0, k0+16).  b[0..1] -> n-tile n0, b[2..3] -> n-tile n0 + 8.
__device__ __forceinline__ void frag_b_nk(uint32_t* b, const bf16* s, int ld, int n0, int k0, int lane) {
  ldsm4(b, s + (size_t)(n0 + (lane & 7) + ((lane >> 4) & 1) * 8) * ld + k0 + ((lane >> 3) & 1) * 8);
}
// B fragments of two n8 tiles where the smem tile is [k][n] (n contiguous): k rows
// [k0, k0+16), n cols [n0, n0+16) -- transposed 8x8 loads.
__device__ __forceinline__ void frag_b_kn(uint32_t* b, const bf16* s, int ld, int k0, int n0, int lane) {
  ldsm4t(b, s + (size_t)(k0 + (lane & 7) + ((lane >> 3) & 1) * 8) * ld + n0 + ((lane >> 4) & 1) * 8);
}

__device__ __forceinline__ float inv_freq(int i, int dh, float theta) {
  return expf(-logf(theta) * (2.0f * (float)i / (float)dh));
}

// rows [r0, r0 + n) of one head's q, k or v (column offset col0 of the [T, 3H] qkv) into a
// bf16 smem tile [n][DH + 8]; rows >= S are zero; RoPE on request.
template <int DH>
__device__ __forceinline__ void load_tile(bf16* dst, const bf16* qkv, int ld_qkv, int b, int S,
                                          int r0, int n, int col0, bool rope, float theta) {
  constexpr int LD = DH + 8;
  if (!rope) {
    for (int e = threadIdx.x; e < n * (DH / 8); e += blockDim.x) {
      const int r = e / (DH / 8), c = (e % (DH / 8)) * 8, s = r0 + r;
      uint4 v = make_uint4(0, 0, 0, 0);
      if (s < S) v = *reinterpret_cast<const uint4*>(qkv + (size_t)(b * S + s) * ld_qkv + col0 + c);
      *reinterpret_cast<uint4*>(dst + r * LD + c) = v;
    }
    return;
  }
  constexpr int HALF = DH / 2;
  for (int e = threadIdx.x; e < n * HALF; e += blockDim.x) {
    const int r = e / HALF, i = e % HALF, s = r0 + r;
    float x1 = 0.f, x2 = 0.f;
    if (s < S) {
      const bf16* src = qkv + (size_t)(b * S + s) * ld_qkv + col0;
      x1 = __bfloat162float(src[i]);
      x2 = __bfloat162float(src[i + HALF]);
    }
    float sn, cs;
    sincosf((float)s * inv_freq(i, DH, theta), &sn, &cs);
    dst[r * LD + i] = __float2bfloat16_rn(x1 * cs - x2 * sn);
    dst[r * LD + i + HALF] = __float2bfloat16_rn(x2 * cs + x1 * sn);
  }
}

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem, bool valid) {
  const uint32_t d = (uint32_t)__cvta_generic_to_shared(smem);
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(d), "l"(gmem), "r"(valid ? 16 : 0)
               : "memory");
}
__device__ __forceinline__ void cp_async4(void* smem, const void* gmem, bool valid) {
  const uint32_t d = (uint32_t)__cvta_generic_to_shared(smem);
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(d), "l"(gmem), "r"(valid ? 4 : 0)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

// Stages rows [r0, r0 + n) of a bf16 [T, ld] matrix at column col0 (DH columns) into a
// [n][DH + 8] smem tile: with RoPE synchronously through load_tile, otherwise as cp.async
// copies (rows >= S zero-filled) that the caller commits and waits for.
template <int DH>
__device__ __forceinline__ void stage_tile(bf16* dst, const bf16* src, int ld, int b, int S, int r0,
                                           int n, int col0, bool rope, float theta) {
  if (rope) {
    load_tile<DH>(dst, src, ld, b, S, r0, n, col0, true, theta);
    return;
  }
  constexpr int LD = DH + 8;
  for (int e = threadIdx.x; e < n * (DH / 8); e += blockDim.x) {
    const int r = e / (DH / 8), c = (e % (DH / 8)) * 8, s = r0 + r;
    const bool ok = s < S;
    cp_async16(dst + r * LD + c, src + (size_t)(b * S + (ok ? s : 0)) * ld + col0 + c, ok);
  }
}

// transpose of the RoPE rotation on accumulator registers: acc[nt][.] holds columns
// nt*8 + 2t (+1) of rows g (c0, c1) and g + 8 (c2, c3); the pair partner of column d < DH/2
// is d + DH/2, i.e. n-tile nt + DH/16 of the same thread.
template <int DH>
__device__ __forceinline__ void rope_bwd_acc(float (&acc)[DH / 8][4], int s0, int s1, int t, float theta) {
#pragma unroll
  for (int nt = 0; nt < DH / 16; ++nt) {
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const int i = nt * 8 + 2 * t + j;
      const float f = inv_freq(i, DH, theta);
      float sn0, cs0, sn1, cs1;
      sincosf((float)s0 * f, &sn0, &cs0);
      sincosf((float)s1 * f, &sn1, &cs1);
      const float d1 = acc[nt][j], d2 = acc[nt + DH / 16][j];
      acc[nt][j] = d1 * cs0 + d2 * sn0;
      acc[nt + DH / 16][j] = d2 * cs0 - d1 * sn0;
      const float e1 = acc[nt][2 + j], e2 = acc[nt + DH / 16][2 + j];
      acc[nt][2 + j] = e1 * cs1 + e2 * sn1;
      acc[nt + DH / 16][2 + j] = e2 * cs1 - e1 * sn1;
    }
  }
}

// ---------------------------------------------------------------------------------------
// RoPE once, in place, on the q and k columns of qkv [T, 3H]: thread = 8 consecutive pair
// indices i of one (token, head); the 8 angles serve both q and k.  The rotated values are
// rounded to bf16 exactly as the staging path rounds them.
// ---------------------------------------------------------------------------------------
template <int DH>
__global__ void __launch_bounds__(256) rope_qk_kernel(bf16* qkv, int T, int S, int n_heads, float theta) {
  pdl_wait();
  pdl_trigger();
  constexpr int HALF = DH / 2, G = HALF / 8;
  const int H = n_heads * DH;
  const int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= (int64_t)T * n_heads * G) return;
  const int gi = (int)(e % G);
  const int64_t th = e / G;
  const int hh = (int)(th % n_heads), tk = (int)(th / n_heads);
  const int s = tk % S, i0 = gi * 8;
  float cs[8], sn[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) sincosf((float)s * inv_freq(i0 + j, DH, theta), &sn[j], &cs[j]);
#pragma unroll
  for (int part = 0; part < 2; ++part) {
    bf16* p = qkv + (size_t)tk * 3 * H + (size_t)part * H + (size_t)hh * DH + i0;
    uint4 u1 = *reinterpret_cast<const uint4*>(p), u2 = *reinterpret_cast<const uint4*>(p + HALF);
    __nv_bfloat16* x1 = reinterpret_cast<__nv_bfloat16*>(&u1);
    __nv_bfloat16* x2 = reinterpret_cast<__nv_bfloat16*>(&u2);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const float a1 = __bfloat162float(x1[j]), a2 = __bfloat162float(x2[j]);
      x1[j] = __float2bfloat16_rn(a1 * cs[j] - a2 * sn[j]);
      x2[j] = __float2bfloat16_rn(a2 * cs[j] + a1 * sn[j]);
    }
    *reinterpret_cast<uint4*>(p) = u1;
    *reinterpret_cast<uint4*>(p + HALF) = u2;
  }
}

// ---------------------------------------------------------------------------------------
// forward: CTA = 64 queries of one (b, head), 4 warps x 16 query rows, 64-key blocks that
// stream through a two-stage ring (block j + 1 is copied while block j is used)
// ---------------------------------------------------------------------------------------
template <int DH>
__global__ void __launch_bounds__(128) attn_fwd_mma_kernel(AttnArgs a) {
  constexpr int LD = DH + 8, NB = 64;
  extern __shared__ __align__(16) uint8_t smraw[];
  bf16* Qs = reinterpret_cast<bf16*>(smraw);
  bf16* KV = Qs + 64 * LD;  // [2 stages][K, V][NB][LD]
  const int bh = blockIdx.y, b = bh / a.n_heads, hh = bh % a.n_heads;
  const int H = a.n_heads * DH, ldq = 3 * H;
  const int q0 = blockIdx.x * 64;
  const bf16* qkv = reinterpret_cast<const bf16*>(a.qkv);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
  const float sl2 = a.scale * kLog2e;
  pdl_wait();
  pdl_trigger();

  const int kend = a.causal ? min(a.S, q0 + 64) : a.S;
  auto stage_kv = [&](int k0, int st) {
    bf16* Kd = KV + (size_t)st * 2 * NB * LD;
    stage_tile<DH>(Kd, qkv, ldq, b, a.S, k0, NB, H + hh * DH, a.rope && !a.qk_rotated, a.rope_theta);
    stage_tile<DH>(Kd + NB * LD, qkv, ldq, b, a.S, k0, NB, 2 * H + hh * DH, false, 0.f);
  };
  stage_tile<DH>(Qs, qkv, ldq, b, a.S, q0, 64, hh * DH, a.rope && !a.qk_rotated, a.rope_theta);
  stage_kv(0, 0);
  cp_async_commit();

  const int qr0 = q0 + warp * 16 + g, qr1 = qr0 + 8;
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
  float o[DH / 8][4];
#pragma unroll
  for (int i = 0; i < DH / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  uint32_t qf[DH / 16][4];

  for (int k0 = 0, it = 0; k0 < kend; k0 += NB, ++it) {
    if (k0 + NB < kend) {
      stage_kv(k0 + NB, (it + 1) & 1);
      cp_async_commit();
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    if (it == 0) {
#pragma unroll
      for (int ks = 0; ks < DH / 16; ++ks) frag_a(qf[ks], Qs, LD, warp * 16, ks * 16, lane);
    }
    const bf16* Ks = KV + (size_t)(it & 1) * 2 * NB * LD;
    const bf16* Vs = Ks + NB * LD;
    float s[NB / 8][4];
#pragma unroll
    for (int i = 0; i < NB / 8; ++i) s[i][0] = s[i][1] = s[i][2] = s[i][3] = 0.f;
#pragma unroll
    for (int ks = 0; ks < DH / 16; ++ks) {
#pragma unroll
      for (int np = 0; np < NB / 16; ++np) {
        uint32_t bb[4];
        frag_b_nk(bb, Ks, LD, np * 16, ks * 16, lane);
        mma16816(s[2 * np], qf[ks], bb[0], bb[1]);
        mma16816(s[2 * np + 1], qf[ks], bb[2], bb[3]);
      }
    }
    // scale, mask, running max
    float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
    for (int nt = 0; nt < NB / 8; ++nt) {
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        const int key = k0 + nt * 8 + 2 * t + j;
        const bool ok = key < a.S;
        s[nt][j] = (ok && (!a.causal || key <= qr0)) ? s[nt][j] * sl2 : -INFINITY;
        s[nt][2 + j] = (ok && (!a.causal || key <= qr1)) ? s[nt][2 + j] * sl2 : -INFINITY;
        mx0 = fmaxf(mx0, s[nt][j]);
        mx1 = fmaxf(mx1, s[nt][2 + j]);
      }
    }
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
    const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
    const float mu0 = mn0 == -INFINITY ? 0.f : mn0, mu1 = mn1 == -INFINITY ? 0.f : mn1;
    const float al0 = exp2f(m0 - mu0), al1 = exp2f(m1 - mu1);
    m0 = mn0;
    m1 = mn1;
    float rs0 = 0.f, rs1 = 0.f;
#pragma unroll
    for (int nt = 0; nt < NB / 8; ++nt) {
      s[nt][0] = exp2f(s[nt][0] - mu0);
      s[nt][1] = exp2f(s[nt][1] - mu0);
      s[nt][2] = exp2f(s[nt][2] - mu1);
      s[nt][3] = exp2f(s[nt][3] - mu1);
      rs0 += s[nt][0] + s[nt][1];
      rs1 += s[nt][2] + s[nt][3];
    }
    rs0 += __shfl_xor_sync(0xffffffffu, rs0, 1);
    rs0 += __shfl_xor_sync(0xffffffffu, rs0, 2);
    rs1 += __shfl_xor_sync(0xffffffffu, rs1, 1);
    rs1 += __shfl_xor_sync(0xffffffffu, rs1, 2);
    l0 = l0 * al0 + rs0;
    l1 = l1 * al1 + rs1;
#pragma unroll
    for (int i = 0; i < DH / 8; ++i) {
      o[i][0] *= al0; o[i][1] *= al0; o[i][2] *= al1; o[i][3] *= al1;
    }
    // O += P V, P from the accumulators (keys k0 + 16kk .. + 15 per A fragment)
#pragma unroll
    for (int kk = 0; kk < NB / 16; ++kk) {
      uint32_t pa[4] = {pk(s[2 * kk][0], s[2 * kk][1]), pk(s[2 * kk][2], s[2 * kk][3]),
                        pk(s[2 * kk + 1][0], s[2 * kk + 1][1]), pk(s[2 * kk + 1][2], s[2 * kk + 1][3])};
#pragma unroll
      for (int np = 0; np < DH / 16; ++np) {
        uint32_t bb[4];
        frag_b_kn(bb, Vs, LD, kk * 16, np * 16, lane);
        mma16816(o[2 * np], pa, bb[0], bb[1]);
        mma16816(o[2 * np + 1], pa, bb[2], bb[3]);
      }
    }
    __syncthreads();  // this stage is refilled by the next iteration's copies
  }
  bf16* O = reinterpret_cast<bf16*>(a.O);
  const float i0 = l0 > 0.f ? 1.f / l0 : 0.f, i1 = l1 > 0.f ? 1.f / l1 : 0.f;
#pragma unroll
  for (int nt = 0; nt < DH / 8; ++nt) {
    const int c = hh * DH + nt * 8 + 2 * t;
    if (qr0 < a.S) *reinterpret_cast<uint32_t*>(O + (size_t)(b * a.S + qr0) * H + c) = pk(o[nt][0] * i0, o[nt][1] * i0);
    if (qr1 < a.S) *reinterpret_cast<uint32_t*>(O + (size_t)(b * a.S + qr1) * H + c) = pk(o[nt][2] * i1, o[nt][3] * i1);
  }
  if (a.lse && t == 0) {
    if (qr0 < a.S) a.lse[(size_t)bh * a.S + qr0] = (m0 + log2f(l0)) * kLn2;
    if (qr1 < a.S) a.lse[(size_t)bh * a.S + qr1] = (m1 + log2f(l1)) * kLn2;
  }
}

// ---------------------------------------------------------------------------------------
// backward dK, dV: CTA = 64 keys of one (b, head) (4 warps x 16 keys); query blocks of QB
// (q, dO, the row log-sum-exp and D) stream through a two-stage ring.  Rows beyond S are
// zero-filled: their q and dO rows are zero, so they add nothing to dK and dV.
// ---------------------------------------------------------------------------------------
template <int DH, int QB>
__global__ void __launch_bounds__(128) attn_bwd_dkdv_mma_kernel(AttnArgs a) {
  constexpr int LD = DH + 8;
  constexpr int STAGE = 2 * QB * LD * 2 + 2 * QB * 4;  // bytes: q, dO, L, D of one block
  extern __shared__ __align__(16) uint8_t smraw[];
  bf16* Ks = reinterpret_cast<bf16*>(smraw);
  bf16* Vs = Ks + 64 * LD;
  uint8_t* ring = reinterpret_cast<uint8_t*>(Vs + 64 * LD);
  const int bh = blockIdx.y, b = bh / a.n_heads, hh = bh % a.n_heads;
  const int H = a.n_heads * DH, ldq = 3 * H;
  const int k0 = blockIdx.x * 64;
  const bf16* qkv = reinterpret_cast<const bf16*>(a.qkv);
  const bf16* dO = reinterpret_cast<const bf16*>(a.dO);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
  const float sl2 = a.scale * kLog2e;
  pdl_wait();
  pdl_trigger();

  stage_tile<DH>(Ks, qkv, ldq, b, a.S, k0, 64, H + hh * DH, a.rope && !a.qk_rotated, a.rope_theta);
  stage_tile<DH>(Vs, qkv, ldq, b, a.S, k0, 64, 2 * H + hh * DH, false, 0.f);
  const int kr0 = k0 + warp * 16 + g, kr1 = kr0 + 8;  // keys of accumulator rows
  float dk[DH / 8][4], dv[DH / 8][4];
#pragma unroll
  for (int i = 0; i < DH / 8; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) dk[i][j] = dv[i][j] = 0.f;

  auto stage_q = [&](int q0, int st) {
    uint8_t* base = ring + (size_t)st * STAGE;
    bf16* Qd = reinterpret_cast<bf16*>(base);
    stage_tile<DH>(Qd, qkv, ldq, b, a.S, q0, QB, hh * DH, a.rope && !a.qk_rotated, a.rope_theta);
    stage_tile<DH>(Qd + QB * LD, dO, H, b, a.S, q0, QB, hh * DH, false, 0.f);
    float* Ld = reinterpret_cast<float*>(Qd + 2 * QB * LD);
    for (int e = threadIdx.x; e < QB; e += blockDim.x) {
      const int s = q0 + e;
      const bool ok = s < a.S;
      cp_async4(Ld + e, a.lse + (size_t)bh * a.S + (ok ? s : 0), ok);
      cp_async4(Ld + QB + e, a.Dscratch + (size_t)bh * a.S + (ok ? s : 0), ok);
    }
  };
  const int qstart = a.causal ? (k0 / QB) * QB : 0;
  stage_q(qstart, 0);
  cp_async_commit();
  for (int q0 = qstart, it = 0; q0 < a.S; q0 += QB, ++it) {
    if (q0 + QB < a.S) {
      stage_q(q0 + QB, (it + 1) & 1);
      cp_async_commit();
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    const bf16* Qs = reinterpret_cast<const bf16*>(ring + (size_t)(it & 1) * STAGE);
    const bf16* Ds_ = Qs + QB * LD;  // dO tile
    const float* Ls = reinterpret_cast<const float*>(Qs + 2 * QB * LD);  // natural-log lse
    const float* Dd = Ls + QB;
    // S^T = K Q^T and dP^T = V dO^T (16 keys x QB queries per warp)
    float st[QB / 8][4], dpt[QB / 8][4];
#pragma unroll
    for (int i = 0; i < QB / 8; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) st[i][j] = dpt[i][j] = 0.f;
#pragma unroll
    for (int ks = 0; ks < DH / 16; ++ks) {
      uint32_t ka[4], va[4];
      frag_a(ka, Ks, LD, warp * 16, ks * 16, lane);
      frag_a(va, Vs, LD, warp * 16, ks * 16, lane);
#pragma unroll
      for (int np = 0; np < QB / 16; ++np) {
        uint32_t bq[4], bo[4];
        frag_b_nk(bq, Qs, LD, np * 16, ks * 16, lane);
        frag_b_nk(bo, Ds_, LD, np * 16, ks * 16, lane);
        mma16816(st[2 * np], ka, bq[0], bq[1]);
        mma16816(st[2 * np + 1], ka, bq[2], bq[3]);
        mma16816(dpt[2 * np], va, bo[0], bo[1]);
        mma16816(dpt[2 * np + 1], va, bo[2], bo[3]);
      }
    }
    // P^T and dS^T (columns are queries)
#pragma unroll
    for (int nt = 0; nt < QB / 8; ++nt) {
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        const int ql = nt * 8 + 2 * t + j, q = q0 + ql;
        const float L = Ls[ql] * kLog2e, Dv = Dd[ql];
        const bool ok0 = kr0 < a.S && (!a.causal || kr0 <= q);
        const bool ok1 = kr1 < a.S && (!a.causal || kr1 <= q);
        const float p0 = ok0 ? exp2f(st[nt][j] * sl2 - L) : 0.f;
        const float p1 = ok1 ? exp2f(st[nt][2 + j] * sl2 - L) : 0.f;
        st[nt][j] = p0;
        st[nt][2 + j] = p1;
        dpt[nt][j] = p0 * (dpt[nt][j] - Dv);
        dpt[nt][2 + j] = p1 * (dpt[nt][2 + j] - Dv);
      }
    }
    // dV += P^T dO ; dK += dS^T Q   (k = queries)
#pragma unroll
    for (int kk = 0; kk < QB / 16; ++kk) {
      uint32_t pa[4] = {pk(st[2 * kk][0], st[2 * kk][1]), pk(st[2 * kk][2], st[2 * kk][3]),
                        pk(st[2 * kk + 1][0], st[2 * kk + 1][1]), pk(st[2 * kk + 1][2], st[2 * kk + 1][3])};
      uint32_t da[4] = {pk(dpt[2 * kk][0], dpt[2 * kk][1]), pk(dpt[2 * kk][2], dpt[2 * kk][3]),
                        pk(dpt[2 * kk + 1][0], dpt[2 * kk + 1][1]), pk(dpt[2 * kk + 1][2], dpt[2 * kk + 1][3])};
#pragma unroll
      for (int np = 0; np < DH / 16; ++np) {
        uint32_t bo[4], bq[4];
        frag_b_kn(bo, Ds_, LD, kk * 16, np * 16, lane);
        frag_b_kn(bq, Qs, LD, kk * 16, np * 16, lane);
        mma16816(dv[2 * np], pa, bo[0], bo[1]);
        mma16816(dv[2 * np + 1], pa, bo[2], bo[3]);
        mma16816(dk[2 * np], da, bq[0], bq[1]);
        mma16816(dk[2 * np + 1], da, bq[2], bq[3]);
      }
    }
    __syncthreads();  // this stage is refilled by the next iteration's copies
  }
#pragma unroll
  for (int i = 0; i < DH / 8; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) dk[i][j] *= a.scale;
  if (a.rope) rope_bwd_acc<DH>(dk, kr0, kr1, t, a.rope_theta);
  bf16* dqkv = reinterpret_cast<bf16*>(a.dqkv);
#pragma unroll
  for (int nt = 0; nt < DH / 8; ++nt) {
    const int c = hh * DH + nt * 8 + 2 * t;
    if (kr0 < a.S) {
      bf16* row = dqkv + (size_t)(b * a.S + kr0) * ldq;
      *reinterpret_cast<uint32_t*>(row + H + c) = pk(dk[nt][0], dk[nt][1]);
      *reinterpret_cast<uint32_t*>(row + 2 * H + c) = pk(dv[nt][0], dv[nt][1]);
    }
    if (kr1 < a.S) {
      bf16* row = dqkv + (size_t)(b * a.S + kr1) * ldq;
      *reinterpret_cast<uint32_t*>(row + H + c) = pk(dk[nt][2], dk[nt][3]);
      *reinterpret_cast<uint32_t*>(row + 2 * H + c) = pk(dv[nt][2], dv[nt][3]);
    }
  }
}

// ---------------------------------------------------------------------------------------
// backward dQ: CTA = 64 queries of one (b, head) (4 warps x 16 queries); 64-key blocks
// streaming through a two-stage ring
// ---------------------------------------------------------------------------------------
template <int DH>
__global__ void __launch_bounds__(128) attn_bwd_dq_mma_kernel(AttnArgs a) {
  constexpr int LD = DH + 8, NB = 64;
  extern __shared__ __align__(16) uint8_t smraw[];
  bf16* Qs = reinterpret_cast<bf16*>(smraw);
  bf16* Os = Qs + 64 * LD;   // dO tile
  bf16* KV = Os + 64 * LD;   // [2 stages][K, V][NB][LD]
  const int bh = blockIdx.y, b = bh / a.n_heads, hh = bh % a.n_heads;
  const int H = a.n_heads * DH, ldq = 3 * H;
  const int q0 = blockIdx.x * 64;
  const bf16* qkv = reinterpret_cast<const bf16*>(a.qkv);
  const bf16* dO = reinterpret_cast<const bf16*>(a.dO);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
  const float sl2 = a.scale * kLog2e;
  pdl_wait();
  pdl_trigger();

  const int kend = a.causal ? min(a.S, q0 + 64) : a.S;
  auto stage_kv = [&](int k0, int st) {
    bf16* Kd = KV + (size_t)st * 2 * NB * LD;
    stage_tile<DH>(Kd, qkv, ldq, b, a.S, k0, NB, H + hh * DH, a.rope && !a.qk_rotated, a.rope_theta);
    stage_tile<DH>(Kd + NB * LD, qkv, ldq, b, a.S, k0, NB, 2 * H + hh * DH, false, 0.f);
  };
  stage_tile<DH>(Qs, qkv, ldq, b, a.S, q0, 64, hh * DH, a.rope && !a.qk_rotated, a.rope_theta);
  stage_tile<DH>(Os, dO, H, b, a.S, q0, 64, hh * DH, false, 0.f);
  stage_kv(0, 0);
  cp_async_commit();
  const int qr0 = q0 + warp * 16 + g, qr1 = qr0 + 8;
  const float L0 = qr0 < a.S ? a.lse[(size_t)bh * a.S + qr0] * kLog2e : INFINITY;
  const float L1 = qr1 < a.S ? a.lse[(size_t)bh * a.S + qr1] * kLog2e : INFINITY;
  const float D0 = qr0 < a.S ? a.Dscratch[(size_t)bh * a.S + qr0] : 0.f;
  const float D1 = qr1 < a.S ? a.Dscratch[(size_t)bh * a.S + qr1] : 0.f;
  float dq[DH / 8][4];
#pragma unroll
  for (int i = 0; i < DH / 8; ++i) dq[i][0] = dq[i][1] = dq[i][2] = dq[i][3] = 0.f;

  for (int k0 = 0, it = 0; k0 < kend; k0 += NB, ++it) {
    if (k0 + NB < kend) {
      stage_kv(k0 + NB, (it + 1) & 1);
      cp_async_commit();
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    const bf16* Ks = KV + (size_t)(it & 1) * 2 * NB * LD;
    const bf16* Vs = Ks + NB * LD;
    float s[NB / 8][4], dp[NB / 8][4];
#pragma unroll
    for (int i = 0; i < NB / 8; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) s[i][j] = dp[i][j] = 0.f;
#pragma unroll
    for (int ks = 0; ks < DH / 16; ++ks) {
      uint32_t qa[4], oa[4];
      frag_a(qa, Qs, LD, warp * 16, ks * 16, lane);
      frag_a(oa, Os, LD, warp * 16, ks * 16, lane);
#pragma unroll
      for (int np = 0; np < NB / 16; ++np) {
        uint32_t bk[4], bv[4];
        frag_b_nk(bk, Ks, LD, np * 16, ks * 16, lane);
        frag_b_nk(bv, Vs, LD, np * 16, ks * 16, lane);
        mma16816(s[2 * np], qa, bk[0], bk[1]);
        mma16816(s[2 * np + 1], qa, bk[2], bk[3]);
        mma16816(dp[2 * np], oa, bv[0], bv[1]);
        mma16816(dp[2 * np + 1], oa, bv[2], bv[3]);
      }
    }
#pragma unroll
    for (int nt = 0; nt < NB / 8; ++nt) {
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        const int key = k0 + nt * 8 + 2 * t + j;
        const bool ok = key < a.S;
        const float p0 = (ok && (!a.causal || key <= qr0)) ? exp2f(s[nt][j] * sl2 - L0) : 0.f;
        const float p1 = (ok && (!a.causal || key <= qr1)) ? exp2f(s[nt][2 + j] * sl2 - L1) : 0.f;
        dp[nt][j] = p0 * (dp[nt][j] - D0);
        dp[nt][2 + j] = p1 * (dp[nt][2 + j] - D1);
      }
    }
    // dQ += dS K   (k = keys)
#pragma unroll
    for (int kk = 0; kk < NB / 16; ++kk) {
      uint32_t da[4] = {pk(dp[2 * kk][0], dp[2 * kk][1]), pk(dp[2 * kk][2], dp[2 * kk][3]),
                        pk(dp[2 * kk + 1][0], dp[2 * kk + 1][1]), pk(dp[2 * kk + 1][2], dp[2 * kk + 1][3])};
#pragma unroll
      for (int np = 0; np < DH / 16; ++np) {
        uint32_t bk[4];
        frag_b_kn(bk, Ks, LD, kk * 16, np * 16, lane);
        mma16816(dq[2 * np], da, bk[0], bk[1]);
        mma16816(dq[2 * np + 1], da, bk[2], bk[3]);
      }
    }
    __syncthreads();  // this stage is refilled by the next iteration's copies
  }
#pragma unroll
  for (int i = 0; i < DH / 8; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) dq[i][j] *= a.scale;
  if (a.rope) rope_bwd_acc<DH>(dq, qr0, qr1, t, a.rope_theta);
  bf16* dqkv = reinterpret_cast<bf16*>(a.dqkv);
#pragma unroll
  for (int nt = 0; nt < DH / 8; ++nt) {
    const int c = hh * DH + nt * 8 + 2 * t;
    if (qr0 < a.S) *reinterpret_cast<uint32_t*>(dqkv + (size_t)(b * a.S + qr0) * ldq + c) = pk(dq[nt][0], dq[nt][1]);
    if (qr1 < a.S) *reinterpret_cast<uint32_t*>(dqkv + (size_t)(b * a.S + qr1) * ldq + c) = pk(dq[nt][2], dq[nt][3]);
  }
}

template <int DH>
cudaError_t fwd(const AttnArgs& a, cudaStream_t st) {
  constexpr int LD = DH + 8;
  const size_t smem = (size_t)5 * 64 * LD * 2;
  auto k = attn_fwd_mma_kernel<DH>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  e = launch_pdl(k, dim3((a.S + 63) / 64, a.B * a.n_heads), dim3(128), smem, st, a);
  note_launch(1);
  return e != cudaSuccess ? e : cudaGetLastError();
}

template <int DH>
cudaError_t bwd(const AttnArgs& a, cudaStream_t st) {
  constexpr int LD = DH + 8, QB = DH == 128 ? 32 : 64;
  const size_t smem1 = (size_t)128 * LD * 2 + 2 * ((size_t)2 * QB * LD * 2 + 2 * QB * 4);
  auto k1 = attn_bwd_dkdv_mma_kernel<DH, QB>;
  cudaError_t e = cudaFuncSetAttribute(k1, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem1);
  if (e != cudaSuccess) return e;
  e = launch_pdl(k1, dim3((a.S + 63) / 64, a.B * a.n_heads), dim3(128), smem1, st, a);
  note_launch(1);
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const size_t smem2 = (size_t)6 * 64 * LD * 2;
  auto k2 = attn_bwd_dq_mma_kernel<DH>;
  e = cudaFuncSetAttribute(k2, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem2);
  if (e != cudaSuccess) return e;
  e = launch_pdl(k2, dim3((a.S + 63) / 64, a.B * a.n_heads), dim3(128), smem2, st, a);
  note_launch(1);
  return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace

bool attention_mma_ok(const AttnArgs& a) {
  return a.dtype == DT_BF16 && (a.head_dim == 64 || a.head_dim == 128);
}

cudaError_t rope_qk_inplace(const AttnArgs& a, cudaStream_t st) {
  if (!attention_mma_ok(a) || !a.rope || a.qk_rotated) return cudaErrorInvalidValue;
  const int T = a.B * a.S;
  const int64_t n = (int64_t)T * a.n_heads * (a.head_dim / 16);
  const unsigned blocks = (unsigned)((n + 255) / 256);
  bf16* qkv = reinterpret_cast<bf16*>(const_cast<void*>(a.qkv));
  const cudaError_t e = a.head_dim == 64
      ? launch_pdl(rope_qk_kernel<64>, dim3(blocks), dim3(256), (size_t)0, st, qkv, T, a.S, a.n_heads, a.rope_theta)
      : launch_pdl(rope_qk_kernel<128>, dim3(blocks), dim3(256), (size_t)0, st, qkv, T, a.S, a.n_heads, a.rope_theta);
  note_launch(1);
  return e != cudaSuccess ? e : cudaGetLastError();
}

// the tcgen05 kernels take every bf16 shape whose q and k are plain or rotated in place:
// the one-block forward for the encoders' short sequences, the block-looping forward for
// longer (the decoder's causal) ones; mma.sync stays for RoPE applied while staging
cudaError_t attention_fwd_mma(const AttnArgs& a, cudaStream_t st) {
  if (attention_tc_ok(a)) return attention_fwd_tc(a, st);
  if (attention_fwd_blocks_tc_ok(a)) return attention_fwd_blocks_tc(a, st);
  return a.head_dim == 64 ? fwd<64>(a, st) : fwd<128>(a, st);
}

// expects D = rowsum(dO * O) already in a.Dscratch
cudaError_t attention_bwd_mma(const AttnArgs& a, cudaStream_t st) {
  if (attention_bwd_tc_ok(a)) return attention_bwd_tc(a, st);
  return a.head_dim == 64 ? bwd<64>(a, st) : bwd<128>(a, st);
}

}  // namespace ra
