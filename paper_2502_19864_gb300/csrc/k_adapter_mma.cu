// k_adapter_mma.cu -- tensor-core (mma.sync m16n8k16, bf16 -> fp32) versions of the adapter
// kernels for the bf16 models.
//
// The adapter (Eq. 1) is a skinny contraction: T x H -> T x m -> T x H with m << H.  Its
// arithmetic (4 T H m flops forward) is beyond what FFMA sustains at HBM speed, while its
// bytes (the T x H input, residual and outputs) make it HBM-bound on tensor cores; so the
// kernels below stream each row tile through shared memory once and fuse everything the
// row needs:
//   forward   z = a W_down; s = GELU(z); v = resid + a + s W_up; LayerNorm (post-LN
//             encoder) or residual stream + RMSNorm (pre-norm decoder) of v;
//   backward  dz = (g W_up^T) * GELU'(z); dh = g + dz W_down^T;
//   dW        per row-chunk partials of dW_up = GELU(z)^T g and dW_down^T = dz^T h, summed
//             afterwards in a fixed order (deterministic).
// CTA = 16 rows x H / 64 warps (64 registers per thread, two CTAs per SM up to H = 1024).
// Phase 1 (the reduction over H) splits K across warps in slices of 64 (128 when the
// partial buffer would pass 64 KB) and sums the per-warp partials of z in a fixed order;
// phase 2 gives each warp 64 of the H output columns; row statistics for the norm are
// combined across warps in shared memory in a fixed order.
#include "common.cuh"
#include "kernels.h"

namespace ra {
namespace {

constexpr int COLS_PER_WARP = 64, R = 16;

__device__ __forceinline__ void mma_bf16(float* d, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
      "{%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void ldsm_x4(uint32_t* r, const void* p) {
  uint32_t a = (uint32_t)__cvta_generic_to_shared(p);
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(a));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t* r, const void* p) {
  uint32_t a = (uint32_t)__cvta_generic_to_shared(p);
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(a));
}
__device__ __forceinline__ void cp_async16(void* smem, const void* gmem, bool valid) {
  const uint32_t s = (uint32_t)__cvta_generic_to_shared(smem);
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(s), "l"(gmem),
               "r"(valid ? 16 : 0)
               : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
}
// B fragments of n8 tile `ntile` (rows 8 ntile .. + 7) for the two k16 steps at k0 (a
// multiple of 32) of a [R, C] bf16 weight in the tiled fragment layout (8 x 32 blocks of 256
// contiguous elements, each row of a block in fragment order): lane l reads elements
// [8 l, 8 l + 8) of the block, 512 contiguous bytes per warp.  .x/.y are b0/b1 of the first
// step, .z/.w of the second.
__device__ __forceinline__ uint4 ld_frag2(const bf16* W, int C, int ntile, int k0, int lane) {
  return __ldg(reinterpret_cast<const uint4*>(W + ((size_t)ntile * (C >> 5) + (k0 >> 5)) * 256 + lane * 8));
}
__device__ __forceinline__ uint32_t pack2(float a, float b) {
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}
__device__ __forceinline__ float2 unpack2(uint32_t u) {
  __nv_bfloat162 h = *reinterpret_cast<__nv_bfloat162*>(&u);
  return __bfloat1622float2(h);
}

// A fragment (16 x 16, row-major in smem, leading dimension ld elements) at (r0, k0)
__device__ __forceinline__ void load_a(uint32_t* a, const bf16* s, int ld, int r0, int k0, int lane) {
  const int r = r0 + (lane & 7) + ((lane >> 3) & 1) * 8;
  const int c = k0 + (lane >> 4) * 8;
  ldsm_x4(a, s + (size_t)r * ld + c);
}

// Phase 1 shared by forward and backward: part[w] = X[16, kslice] * Bw^T over this warp's
// slice [kbase, kbase + ks_len) of H, where Bw is [m, H] bf16 in the tiled fragment layout (B
// fragments read directly, 16 bytes per thread per two k16 steps; the matrix is small and
// stays in L1/L2).  The m output columns
// are produced in groups of 8 n-tiles to bound the registers.  Rows of part are MB + 8 floats
// apart, so the float2 stores of one half-warp fall in distinct banks.
template <int MB>
__device__ __forceinline__ void phase1_store(const bf16* Xs, int ldx, const bf16* Bw, int H,
                                             int kbase, int ks_len, float* part, int lane) {
  const int g = lane >> 2, t = lane & 3;
  constexpr int NG = MB >= 64 ? MB / 64 : 1, NTG = MB >= 64 ? 8 : MB / 8;
#pragma unroll 1
  for (int ng = 0; ng < NG; ++ng) {
    float acc[NTG][4];
#pragma unroll
    for (int nt = 0; nt < NTG; ++nt) acc[nt][0] = acc[nt][1] = acc[nt][2] = acc[nt][3] = 0.f;
#pragma unroll 1
    for (int k0 = kbase; k0 < kbase + ks_len; k0 += 32) {
      uint32_t a0[4], a1[4];
      load_a(a0, Xs, ldx, 0, k0, lane);
      load_a(a1, Xs, ldx, 0, k0 + 16, lane);
#pragma unroll
      for (int nt = 0; nt < NTG; ++nt) {
        const uint4 b = ld_frag2(Bw, H, ng * 8 + nt, k0, lane);
        mma_bf16(acc[nt], a0, b.x, b.y);
        mma_bf16(acc[nt], a1, b.z, b.w);
      }
    }
#pragma unroll
    for (int nt = 0; nt < NTG; ++nt) {
      const int c = ng * 64 + nt * 8 + 2 * t;
      *reinterpret_cast<float2*>(part + g * (MB + 8) + c) = make_float2(acc[nt][0], acc[nt][1]);
      *reinterpret_cast<float2*>(part + (g + 8) * (MB + 8) + c) = make_float2(acc[nt][2], acc[nt][3]);
    }
  }
}

// K-slice of phase 1: 64 columns of H per warp unless the per-warp partials of z would pass
// 64 KB of shared memory, then 128 (and only the first H / 128 warps take part)
__host__ __device__ inline int phase1_slice(int H, int m) {
  return (H / 64) * R * m * 4 > 65536 ? 128 : 64;
}

// Phase 2: acc[16 rows, this warp's 64 columns] = S[16, m] * Bn^T where Bn is [H, m] bf16
// in the tiled fragment layout (n = output column, k = bottleneck index).
template <int MB>
__device__ __forceinline__ void phase2(float (&acc)[8][4], const bf16* Ss, int lds,
                                       const bf16* Bn, int m, int nbase, int lane) {
#pragma unroll
  for (int nt = 0; nt < 8; ++nt) acc[nt][0] = acc[nt][1] = acc[nt][2] = acc[nt][3] = 0.f;
#pragma unroll
  for (int k0 = 0; k0 < MB; k0 += 32) {
    uint32_t a0[4], a1[4];
    load_a(a0, Ss, lds, 0, k0, lane);
    load_a(a1, Ss, lds, 0, k0 + 16, lane);
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      const uint4 b = ld_frag2(Bn, m, (nbase >> 3) + nt, k0, lane);
      mma_bf16(acc[nt], a0, b.x, b.y);
      mma_bf16(acc[nt], a1, b.z, b.w);
    }
  }
}

struct FwdArgs {
  int T, H, m;
  const bf16* a;          // [T, H]
  const bf16* WdT;        // [m, H]
  const bf16* WuT;        // [H, m]
  float* z;               // [T, m] or null
  const void* resid;      // encoder bf16, decoder f32
  const float* gamma;
  const float* beta;
  float eps;
  bf16* y;                // normalised output
  float* x_out;           // decoder residual stream out
  bf16* xhat;             // encoder, nullable
  float* rstd;            // nullable
  bool stage_gb;          // gamma (and beta) staged in shared memory
};

// Issues cp.async copies of R rows of a bf16 [T, H] matrix into smem (ld = H + 8); rows >= T
// are zero-filled.  The caller waits (cp_async_wait_all) and synchronises.
__device__ __forceinline__ void load_rows_bf16_async(bf16* dst, int ld, const bf16* src, int t0, int T,
                                                     int H, int R) {
  const int vec = H / 8;
  for (int e = threadIdx.x; e < R * vec; e += blockDim.x) {
    const int r = e / vec, c = (e % vec) * 8;
    const bool ok = t0 + r < T;
    cp_async16(dst + (size_t)r * ld + c, src + (size_t)(ok ? t0 + r : 0) * H + c, ok);
  }
}
__device__ __forceinline__ void load_rows_f32_as_bf16(bf16* dst, int ld, const float* src, int t0,
                                                      int T, int H, int R) {
  const int vec = H / 4, n = R * vec, step = blockDim.x;
  // up to eight 16-byte loads in flight per thread before any conversion
  for (int e0 = threadIdx.x; e0 < n; e0 += 8 * step) {
    float4 v[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const int e = e0 + k * step, r = e / vec, c = (e % vec) * 4;
      v[k] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (e < n && t0 + r < T) v[k] = __ldg(reinterpret_cast<const float4*>(src + (size_t)(t0 + r) * H + c));
    }
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const int e = e0 + k * step, r = e / vec, c = (e % vec) * 4;
      if (e < n)
        *reinterpret_cast<uint2*>(dst + (size_t)r * ld + c) = make_uint2(pack2(v[k].x, v[k].y), pack2(v[k].z, v[k].w));
    }
  }
}

// Thread-count classes (H / 64 warps): SZ 0 for H <= 768 (two CTAs per SM at 85 registers),
// SZ 1 for H <= 1024 (two CTAs per SM at 64), SZ 2 above (one CTA per SM, 64 registers).
#define RA_ROWS_BOUNDS(SZ) __launch_bounds__((SZ) == 0 ? 384 : (SZ) == 1 ? 512 : 1024, (SZ) == 2 ? 1 : 2)
__host__ __device__ constexpr int size_class(int H) { return H <= 768 ? 0 : H <= 1024 ? 1 : 2; }

// Shared-memory layout of the forward kernel (byte offsets):
//   [0, part)       a rows [R][H + 8] bf16; after the norm, the output y of each warp's columns
//   [part, s)       per-warp partials of z [W1][R][MB + 8] f32; once z is summed (encoder) the
//                   residual rows [R][H + 8] bf16, then xhat of each warp's columns
//   [s, stat)       GELU(z) [R][MB + 8] bf16
//   [stat, gb)      per-warp row summaries [W][16] float2
//   [gb, bytes)     gamma (and beta) staged at the start, when they fit without costing a CTA
struct FwdLayout { int part, s, stat, gb, bytes; };
__host__ __device__ inline FwdLayout fwd_layout(int H, int m, int gb_floats) {
  const int W = H / COLS_PER_WARP, W1 = H / phase1_slice(H, m);
  const int zpart = W1 * R * (m + 8) * 4, rows = R * (H + 8) * 2;
  FwdLayout L;
  L.part = rows;
  L.s = L.part + (zpart > rows ? zpart : rows);
  L.stat = L.s + R * (m + 8) * 2;
  L.gb = L.stat + W * 16 * 8;
  L.bytes = L.gb + gb_floats * 4;
  return L;
}

// cp.async of the 16 x 64 block of rows [t0, t0 + 16) and this warp's columns [c0, c0 + 64)
// of a bf16 [T, H] matrix (rows >= T zero-filled); four 16-byte copies per lane
__device__ __forceinline__ void load_block_async(bf16* dst, int ld, const bf16* src, int t0, int T,
                                                 int H, int c0, int lane) {
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int e = lane + 32 * i, r = e >> 3, c = c0 + (e & 7) * 8;
    const bool ok = t0 + r < T;
    cp_async16(dst + (size_t)r * ld + c, src + (size_t)(ok ? t0 + r : 0) * H + c, ok);
  }
}
// copies the warp's 16 x 64 block from shared memory to rows [t0, t0 + 16) of a bf16 [T, H]
// matrix: every store instruction writes four whole 128-byte row segments
__device__ __forceinline__ void store_block(bf16* dst, int H, const bf16* src, int ld, int t0, int T,
                                            int c0, int lane) {
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int e = lane + 32 * i, r = e >> 3, c = c0 + (e & 7) * 8;
    if (t0 + r < T)
      *reinterpret_cast<uint4*>(dst + (size_t)(t0 + r) * H + c) = *reinterpret_cast<const uint4*>(src + (size_t)r * ld + c);
  }
}

// MODE: FWD_LN (post-LN encoder: residual add, LayerNorm), FWD_RMS (pre-norm decoder: f32
// residual stream, RMSNorm of it), FWD_NONE (the paper's post-FFN placement: y = a +
// GELU(a W_down) W_up, no residual operand, no norm)
enum : int { FWD_LN = 0, FWD_RMS = 1, FWD_NONE = 2 };

template <int MB, int MODE, int SZ>
__global__ void RA_ROWS_BOUNDS(SZ) adapter_fwd_mma_kernel(FwdArgs p) {
  constexpr bool DEC = MODE == FWD_RMS;
  extern __shared__ __align__(16) uint8_t sm[];
  pdl_wait();
  pdl_trigger();
  const int H = p.H, W = H / COLS_PER_WARP;
  const int KS = phase1_slice(H, MB), W1 = H / KS;
  const int lda = H + 8, lds = MB + 8;
  const FwdLayout L = fwd_layout(H, MB, 0);
  bf16* As = reinterpret_cast<bf16*>(sm);
  float* part = reinterpret_cast<float*>(sm + L.part);
  bf16* Rs = reinterpret_cast<bf16*>(sm + L.part);
  bf16* Ss = reinterpret_cast<bf16*>(sm + L.s);
  float2* stat = reinterpret_cast<float2*>(sm + L.stat);
  float* gbs = reinterpret_cast<float*>(sm + L.gb);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, t = lane & 3;
  const int t0 = blockIdx.x * R;
  const int nbase = warp * COLS_PER_WARP;

  load_rows_bf16_async(As, lda, p.a, t0, p.T, H, R);
  if (p.stage_gb) {
    const int nv = (DEC ? 1 : 2) * (H / 4);
    for (int e = threadIdx.x; e < nv; e += blockDim.x) {
      const float* src = e < H / 4 ? p.gamma + 4 * e : p.beta + 4 * (e - H / 4);
      cp_async16(gbs + 4 * e, src, true);
    }
  }
  cp_async_wait_all();
  __syncthreads();
  if (warp < W1) phase1_store<MB>(As, lda, p.WdT, H, warp * KS, KS, part + (size_t)warp * R * (MB + 8), lane);
  __syncthreads();
  for (int e = threadIdx.x; e < R * MB; e += blockDim.x) {
    const int r = e / MB, j = e % MB;
    float zs = 0.f;
    for (int w = 0; w < W1; ++w) zs += part[((size_t)w * R + r) * (MB + 8) + j];
    if (p.z && t0 + r < p.T) p.z[(size_t)(t0 + r) * MB + j] = zs;
    Ss[r * lds + j] = __float2bfloat16_rn(gelu_f(zs));
  }
  __syncthreads();
  // encoder: the residual rows of this warp's columns land in the (now free) partial buffer
  // while phase 2 runs
  if (MODE == FWD_LN) load_block_async(Rs, lda, reinterpret_cast<const bf16*>(p.resid), t0, p.T, H, nbase, lane);
  float v[8][4];
  phase2<MB>(v, Ss, lds, p.WuT, MB, nbase, lane);
  if (MODE == FWD_LN) {
    cp_async_wait_all();
    __syncwarp();
  }
  if (MODE == FWD_NONE) {
    // y = a + GELU(z) W_up, through this warp's columns of the a rows
    const int rl0 = g, rl1 = g + 8;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      const int c = nbase + nt * 8 + 2 * t;
      const float2 a0 = unpack2(*reinterpret_cast<const uint32_t*>(As + (size_t)rl0 * lda + c));
      const float2 a1 = unpack2(*reinterpret_cast<const uint32_t*>(As + (size_t)rl1 * lda + c));
      *reinterpret_cast<uint32_t*>(As + (size_t)rl0 * lda + c) = pack2(v[nt][0] + a0.x, v[nt][1] + a0.y);
      *reinterpret_cast<uint32_t*>(As + (size_t)rl1 * lda + c) = pack2(v[nt][2] + a1.x, v[nt][3] + a1.y);
    }
    __syncwarp();
    store_block(p.y, H, As, lda, t0, p.T, nbase, lane);
    return;
  }
  const int rl0 = g, rl1 = g + 8;  // local rows of c0/c1 and c2/c3
  const int r0 = t0 + rl0, r1 = t0 + rl1;
  float s0 = 0.f, s1 = 0.f;
#pragma unroll
  for (int nt = 0; nt < 8; ++nt) {
    const int c = nbase + nt * 8 + 2 * t;
    float2 a0 = unpack2(*reinterpret_cast<const uint32_t*>(As + (size_t)rl0 * lda + c));
    float2 a1 = unpack2(*reinterpret_cast<const uint32_t*>(As + (size_t)rl1 * lda + c));
    float2 q0 = make_float2(0.f, 0.f), q1 = make_float2(0.f, 0.f);
    if (DEC) {
      const float* rs = reinterpret_cast<const float*>(p.resid);
      if (r0 < p.T) q0 = *reinterpret_cast<const float2*>(rs + (size_t)r0 * H + c);
      if (r1 < p.T) q1 = *reinterpret_cast<const float2*>(rs + (size_t)r1 * H + c);
    } else {
      q0 = unpack2(*reinterpret_cast<const uint32_t*>(Rs + (size_t)rl0 * lda + c));
      q1 = unpack2(*reinterpret_cast<const uint32_t*>(Rs + (size_t)rl1 * lda + c));
    }
    v[nt][0] += a0.x + q0.x; v[nt][1] += a0.y + q0.y;
    v[nt][2] += a1.x + q1.x; v[nt][3] += a1.y + q1.y;
    if (DEC) {
      s0 += v[nt][0] * v[nt][0] + v[nt][1] * v[nt][1];
      s1 += v[nt][2] * v[nt][2] + v[nt][3] * v[nt][3];
    } else {
      s0 += v[nt][0] + v[nt][1];
      s1 += v[nt][2] + v[nt][3];
    }
  }
  s0 += __shfl_xor_sync(0xffffffffu, s0, 1);
  s0 += __shfl_xor_sync(0xffffffffu, s0, 2);
  s1 += __shfl_xor_sync(0xffffffffu, s1, 1);
  s1 += __shfl_xor_sync(0xffffffffu, s1, 2);
  // Row statistics with one barrier.  Each warp publishes a summary of its 64 columns of the
  // 16 rows; after the barrier lanes 0-15 of every warp merge the W summaries of one row in
  // warp order (the same order in every warp) and the quads fetch their two rows by shuffle.
  //   RMSNorm:   the sum of squares;
  //   LayerNorm: the mean and the centred sum of squares of the 64 columns, merged with the
  //              pairwise update of Chan, Golub and LeVeque for equal counts,
  //              M2 = sum_w M2_w + 64 sum_w (mean_w - mean)^2.
  float mu0 = 0.f, mu1 = 0.f;
  if (!DEC) {
    mu0 = s0 * (1.f / COLS_PER_WARP);
    mu1 = s1 * (1.f / COLS_PER_WARP);
    s0 = s1 = 0.f;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      const float d0 = v[nt][0] - mu0, d1 = v[nt][1] - mu0, d2 = v[nt][2] - mu1, d3 = v[nt][3] - mu1;
      s0 += d0 * d0 + d1 * d1;
      s1 += d2 * d2 + d3 * d3;
    }
    s0 += __shfl_xor_sync(0xffffffffu, s0, 1);
    s0 += __shfl_xor_sync(0xffffffffu, s0, 2);
    s1 += __shfl_xor_sync(0xffffffffu, s1, 1);
    s1 += __shfl_xor_sync(0xffffffffu, s1, 2);
  }
  if (t == 0) {
    stat[warp * 16 + rl0] = make_float2(mu0, s0);
    stat[warp * 16 + rl1] = make_float2(mu1, s1);
  }
  __syncthreads();
  float mean = 0.f, rstd = 0.f;
  if (lane < 16) {
    if (DEC) {
      float q = 0.f;
      for (int w = 0; w < W; ++w) q += stat[w * 16 + lane].y;
      rstd = rsqrtf(q / H + p.eps);
    } else {
      float sm = 0.f;
      for (int w = 0; w < W; ++w) sm += stat[w * 16 + lane].x;
      mean = sm / W;
      float q = 0.f, dd = 0.f;
      for (int w = 0; w < W; ++w) {
        const float2 st = stat[w * 16 + lane];
        const float d = st.x - mean;
        q += st.y;
        dd += d * d;
      }
      rstd = rsqrtf((q + COLS_PER_WARP * dd) / H + p.eps);
    }
  }
  const float rs0 = __shfl_sync(0xffffffffu, rstd, rl0), rs1 = __shfl_sync(0xffffffffu, rstd, rl1);
  const float* gam = p.stage_gb ? gbs : p.gamma;
  if (DEC) {
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      const int c = nbase + nt * 8 + 2 * t;
      const float2 gm = *reinterpret_cast<const float2*>(gam + c);
      if (r0 < p.T) *reinterpret_cast<float2*>(p.x_out + (size_t)r0 * H + c) = make_float2(v[nt][0], v[nt][1]);
      if (r1 < p.T) *reinterpret_cast<float2*>(p.x_out + (size_t)r1 * H + c) = make_float2(v[nt][2], v[nt][3]);
      // y goes through this warp's columns of the a rows (read above by this thread only)
      *reinterpret_cast<uint32_t*>(As + (size_t)rl0 * lda + c) = pack2(v[nt][0] * rs0 * gm.x, v[nt][1] * rs0 * gm.y);
      *reinterpret_cast<uint32_t*>(As + (size_t)rl1 * lda + c) = pack2(v[nt][2] * rs1 * gm.x, v[nt][3] * rs1 * gm.y);
    }
    __syncwarp();
    store_block(p.y, H, As, lda, t0, p.T, nbase, lane);
  } else {
    const float m0 = __shfl_sync(0xffffffffu, mean, rl0), m1 = __shfl_sync(0xffffffffu, mean, rl1);
    const float* bet = p.stage_gb ? gbs + H : p.beta;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      const int c = nbase + nt * 8 + 2 * t;
      const float2 gm = *reinterpret_cast<const float2*>(gam + c);
      const float2 bt = *reinterpret_cast<const float2*>(bet + c);
      const float x00 = (v[nt][0] - m0) * rs0, x01 = (v[nt][1] - m0) * rs0;
      const float x10 = (v[nt][2] - m1) * rs1, x11 = (v[nt][3] - m1) * rs1;
      // y and xhat go through this warp's columns of the a rows and of the residual rows
      *reinterpret_cast<uint32_t*>(As + (size_t)rl0 * lda + c) = pack2(x00 * gm.x + bt.x, x01 * gm.y + bt.y);
      *reinterpret_cast<uint32_t*>(As + (size_t)rl1 * lda + c) = pack2(x10 * gm.x + bt.x, x11 * gm.y + bt.y);
      *reinterpret_cast<uint32_t*>(Rs + (size_t)rl0 * lda + c) = pack2(x00, x01);
      *reinterpret_cast<uint32_t*>(Rs + (size_t)rl1 * lda + c) = pack2(x10, x11);
    }
    __syncwarp();
    store_block(p.y, H, As, lda, t0, p.T, nbase, lane);
    if (p.xhat) store_block(p.xhat, H, Rs, lda, t0, p.T, nbase, lane);
  }
  if (p.rstd && warp == 0 && t == 0) {
    if (r0 < p.T) p.rstd[r0] = rs0;
    if (r1 < p.T) p.rstd[r1] = rs1;
  }
}

// ---------------------------------------------------------------------------------------
// backward rows: dz = (g W_up^T) * GELU'(z); dh = g + dz W_down^T
// ---------------------------------------------------------------------------------------
struct BwdArgs {
  int T, H, m;
  const float* g;     // [T, H]
  const float* z;     // [T, m]
  const bf16* Wu;     // [m, H]
  const bf16* Wd;     // [H, m]
  float* dz;          // [T, m] f32 of scratch, used as [T, m] bf16 GELU(z) then [T, m] bf16 dz
  void* dh;           // [T, H] or null: bf16, or f32 when DH_F32
};

template <int MB, int SZ, bool DH_F32>
__global__ void RA_ROWS_BOUNDS(SZ) adapter_bwd_rows_mma_kernel(BwdArgs p) {
  extern __shared__ __align__(16) uint8_t sm[];
  pdl_wait();
  pdl_trigger();
  const int H = p.H;
  const int KS = phase1_slice(H, MB), W1 = H / KS;
  const int ldg = H + 8, lds = MB + 8;
  bf16* Gs = reinterpret_cast<bf16*>(sm);
  float* part = reinterpret_cast<float*>(Gs + (size_t)R * ldg);
  bf16* Ds = reinterpret_cast<bf16*>(part + (size_t)W1 * R * (MB + 8));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, t = lane & 3;
  const int t0 = blockIdx.x * R;

  load_rows_f32_as_bf16(Gs, ldg, p.g, t0, p.T, H, R);
  __syncthreads();
  if (warp < W1) phase1_store<MB>(Gs, ldg, p.Wu, H, warp * KS, KS, part + (size_t)warp * R * (MB + 8), lane);
  __syncthreads();
  // the weight-gradient kernel reads GELU(z) and dz as the bf16 operands it multiplies: both
  // leave here rounded once, in the dz buffer ([T][m] GELU(z), then [T][m] dz)
  bf16* sz = reinterpret_cast<bf16*>(p.dz);
  bf16* dzb = sz + (size_t)p.T * MB;
  for (int e = threadIdx.x; e < R * MB; e += blockDim.x) {
    const int r = e / MB, j = e % MB;
    float ds = 0.f;
    for (int w = 0; w < W1; ++w) ds += part[((size_t)w * R + r) * (MB + 8) + j];
    float dz = 0.f;
    const bf16 d16 = __float2bfloat16_rn(0.f);
    bf16 dzr = d16;
    if (t0 + r < p.T) {
      const float zz = p.z[(size_t)(t0 + r) * MB + j];
      dz = ds * gelu_grad_f(zz);
      dzr = __float2bfloat16_rn(dz);
      sz[(size_t)(t0 + r) * MB + j] = __float2bfloat16_rn(gelu_f(zz));
      dzb[(size_t)(t0 + r) * MB + j] = dzr;
    }
    Ds[r * lds + j] = dzr;
  }
  if (!p.dh) return;
  __syncthreads();
  const int nbase = warp * COLS_PER_WARP;
  float v[8][4];
  phase2<MB>(v, Ds, lds, p.Wd, MB, nbase, lane);
  const int r0 = t0 + g, r1 = r0 + 8;
  if (DH_F32) {
    // fp32 dh (the gradient feeding a LayerNorm backward), written from registers
    float* dh = reinterpret_cast<float*>(p.dh);
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      const int c = nbase + nt * 8 + 2 * t;
      if (r0 < p.T) {
        const float2 q0 = *reinterpret_cast<const float2*>(p.g + (size_t)r0 * H + c);
        *reinterpret_cast<float2*>(dh + (size_t)r0 * H + c) = make_float2(v[nt][0] + q0.x, v[nt][1] + q0.y);
      }
      if (r1 < p.T) {
        const float2 q1 = *reinterpret_cast<const float2*>(p.g + (size_t)r1 * H + c);
        *reinterpret_cast<float2*>(dh + (size_t)r1 * H + c) = make_float2(v[nt][2] + q1.x, v[nt][3] + q1.y);
      }
    }
    return;
  }
  // dh goes through this warp's columns of the staged g rows, then out in whole row segments
#pragma unroll
  for (int nt = 0; nt < 8; ++nt) {
    const int c = nbase + nt * 8 + 2 * t;
    float2 q0 = make_float2(0.f, 0.f), q1 = make_float2(0.f, 0.f);
    if (r0 < p.T) q0 = *reinterpret_cast<const float2*>(p.g + (size_t)r0 * H + c);
    if (r1 < p.T) q1 = *reinterpret_cast<const float2*>(p.g + (size_t)r1 * H + c);
    *reinterpret_cast<uint32_t*>(Gs + (size_t)g * ldg + c) = pack2(v[nt][0] + q0.x, v[nt][1] + q0.y);
    *reinterpret_cast<uint32_t*>(Gs + (size_t)(g + 8) * ldg + c) = pack2(v[nt][2] + q1.x, v[nt][3] + q1.y);
  }
  __syncwarp();
  store_block(reinterpret_cast<bf16*>(p.dh), H, Gs, ldg, t0, p.T, nbase, lane);
}

// ---------------------------------------------------------------------------------------
// dW partials over a chunk of rows, 64 columns of H per CTA:
//   pWu[c][j][i]  = sum_t GELU(z[t, j]) g[t, i]
//   pWdT[c][j][i] = sum_t dz[t, j] h[t, i]
// 8 warps: warps 0-3 -> dW_up, 4-7 -> dW_down^T; warp owns m/4 bottleneck rows x 64 cols.
// ---------------------------------------------------------------------------------------
struct DwArgs {
  int T, H, m, chunk;
  const float* g;
  const bf16* h;
  const bf16* s;    // GELU(z) [T, m], bf16
  const bf16* dz;   // dz [T, m], bf16
  float* partials;
};

constexpr int DWC = 64, DWR = 32;

template <int MB>
__global__ void __launch_bounds__(256) adapter_dw_mma_kernel(DwArgs p) {
  pdl_wait();
  pdl_trigger();
  // 4 warps per output matrix: with m >= 64 each owns m/64 tiles of 16 bottleneck rows and
  // all 64 columns; with m = 32 each owns one 16-row tile and one 32-column half
  constexpr int LDJ = MB + 8, LDI = DWC + 8;
  constexpr int MTW = MB >= 64 ? MB / 64 : 1;
  constexpr int NPW = MB >= 64 ? 4 : 2;  // pairs of n8 tiles per warp
  __shared__ __align__(16) bf16 Ssm[DWR * LDJ], Dsm[DWR * LDJ], Gsm[DWR * LDI], Hsm[DWR * LDI];
  const int H = p.H, i0 = blockIdx.x * DWC, c = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, t = lane & 3;
  const int which = warp >> 2;                    // 0: dW_up, 1: dW_down^T
  const int jbase = MB >= 64 ? (warp & 3) * (MB / 4) : ((warp & 3) & 1) * 16;
  const int ibase = MB >= 64 ? 0 : ((warp & 3) >> 1) * 32;
  const int tb = c * p.chunk, te = min(p.T, tb + p.chunk);
  float acc[MTW][2 * NPW][4];
#pragma unroll
  for (int a = 0; a < MTW; ++a)
#pragma unroll
    for (int nt = 0; nt < 2 * NPW; ++nt)
#pragma unroll
      for (int i = 0; i < 4; ++i) acc[a][nt][i] = 0.f;
  const bf16* X = which ? Dsm : Ssm;
  const bf16* Y = which ? Hsm : Gsm;
  // each thread's share of one 32-row tile: (GELU(z), dz) pairs and (g, h) quads
  constexpr int NZ = DWR * (MB / 2) / 256, NG = DWR * (DWC / 4) / 256;
  uint32_t zr[NZ], dr[NZ];
  float4 gr[NG];
  uint2 hr[NG];
  auto fetch = [&](int r0) {
#pragma unroll
    for (int q = 0; q < NZ; ++q) {
      const int e = threadIdx.x + q * 256, r = e / (MB / 2), j = (e % (MB / 2)) * 2, tt = r0 + r;
      zr[q] = dr[q] = 0u;
      if (tt < te) {
        zr[q] = *reinterpret_cast<const uint32_t*>(p.s + (size_t)tt * MB + j);
        dr[q] = *reinterpret_cast<const uint32_t*>(p.dz + (size_t)tt * MB + j);
      }
    }
#pragma unroll
    for (int q = 0; q < NG; ++q) {
      const int e = threadIdx.x + q * 256, r = e / (DWC / 4), i = (e % (DWC / 4)) * 4, tt = r0 + r;
      gr[q] = make_float4(0.f, 0.f, 0.f, 0.f);
      hr[q] = make_uint2(0, 0);
      if (tt < te) {
        gr[q] = *reinterpret_cast<const float4*>(p.g + (size_t)tt * H + i0 + i);
        hr[q] = *reinterpret_cast<const uint2*>(p.h + (size_t)tt * H + i0 + i);
      }
    }
  };
  if (tb < te) fetch(tb);
  for (int r0 = tb; r0 < te; r0 += DWR) {
    __syncthreads();
#pragma unroll
    for (int q = 0; q < NZ; ++q) {
      const int e = threadIdx.x + q * 256, r = e / (MB / 2), j = (e % (MB / 2)) * 2;
      *reinterpret_cast<uint32_t*>(Ssm + r * LDJ + j) = zr[q];
      *reinterpret_cast<uint32_t*>(Dsm + r * LDJ + j) = dr[q];
    }
#pragma unroll
    for (int q = 0; q < NG; ++q) {
      const int e = threadIdx.x + q * 256, r = e / (DWC / 4), i = (e % (DWC / 4)) * 4;
      *reinterpret_cast<uint2*>(Gsm + r * LDI + i) = make_uint2(pack2(gr[q].x, gr[q].y), pack2(gr[q].z, gr[q].w));
      *reinterpret_cast<uint2*>(Hsm + r * LDI + i) = hr[q];
    }
    __syncthreads();
    if (r0 + DWR < te) fetch(r0 + DWR);  // next tile's loads overlap this tile's products
#pragma unroll
    for (int ks = 0; ks < DWR / 16; ++ks) {
      const int k0 = ks * 16;
      // A = X^T (rows j, cols t): transposed 8x8 loads of X[t][j]
      uint32_t a[MTW][4];
#pragma unroll
      for (int mtw = 0; mtw < MTW; ++mtw) {
        const int j0 = jbase + mtw * 16;
        const int mat = lane >> 3, rr = lane & 7;
        const int trow = k0 + rr + (mat >> 1) * 8, jcol = j0 + (mat & 1) * 8;
        ldsm_x4_t(a[mtw], X + trow * LDJ + jcol);
      }
      // B = Y[t][i] (k = t, n = i): transposed 8x8 loads give the column-major fragments
#pragma unroll
      for (int np = 0; np < NPW; ++np) {
        uint32_t b[4];
        const int mat = lane >> 3, rr = lane & 7;
        const int trow = k0 + rr + (mat & 1) * 8, icol = ibase + np * 16 + (mat >> 1) * 8;
        ldsm_x4_t(b, Y + trow * LDI + icol);
#pragma unroll
        for (int mtw = 0; mtw < MTW; ++mtw) {
          mma_bf16(acc[mtw][2 * np], a[mtw], b[0], b[1]);
          mma_bf16(acc[mtw][2 * np + 1], a[mtw], b[2], b[3]);
        }
      }
    }
  }
  float* out = p.partials + (size_t)c * 2 * H * MB + (which ? (size_t)H * MB : 0);
#pragma unroll
  for (int mtw = 0; mtw < MTW; ++mtw)
#pragma unroll
    for (int nt = 0; nt < 2 * NPW; ++nt) {
      const int j = jbase + mtw * 16 + g, i = i0 + ibase + nt * 8 + 2 * t;
      *reinterpret_cast<float2*>(out + (size_t)j * H + i) = make_float2(acc[mtw][nt][0], acc[mtw][nt][1]);
      *reinterpret_cast<float2*>(out + (size_t)(j + 8) * H + i) = make_float2(acc[mtw][nt][2], acc[mtw][nt][3]);
    }
}

// shared memory of the backward row kernel
size_t rows_smem(int H, int m) {
  const int W = H / COLS_PER_WARP, W1 = H / phase1_slice(H, m);
  return (size_t)R * (H + 8) * 2 + (size_t)W1 * R * (m + 8) * 4 + (size_t)R * (m + 8) * 2 + (W * 16 + 16) * 4;
}

int smem_per_sm() {
  static int v = -1;
  if (v < 0) {
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) == cudaSuccess &&
        cudaDeviceGetAttribute(&n, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev) == cudaSuccess)
      v = n;
    else
      v = 0;
  }
  return v;
}

template <int MB, int MODE>
cudaError_t launch_fwd(FwdArgs p, cudaStream_t st) {
  constexpr bool DEC = MODE == FWD_RMS;
  // gamma (and beta) go to shared memory when that keeps the CTAs per SM (1 KB reserved each)
  const int gbf = MODE == FWD_NONE ? 0 : (DEC ? 1 : 2) * p.H;
  const size_t s0 = fwd_layout(p.H, MB, 0).bytes, s1 = fwd_layout(p.H, MB, gbf).bytes;
  const int per_sm = smem_per_sm();
  const bool aligned = MODE != FWD_NONE && ((uintptr_t)p.gamma & 15) == 0 &&
                       (DEC || ((uintptr_t)p.beta & 15) == 0);
  p.stage_gb = aligned && s1 <= 220 * 1024 && per_sm > 0 &&
               per_sm / (int)(s1 + 1024) == per_sm / (int)(s0 + 1024);
  const size_t smem = p.stage_gb ? s1 : s0;
  const int sz = size_class(p.H);
  auto k = sz == 0 ? adapter_fwd_mma_kernel<MB, MODE, 0>
         : sz == 1 ? adapter_fwd_mma_kernel<MB, MODE, 1> : adapter_fwd_mma_kernel<MB, MODE, 2>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  e = launch_pdl(k, dim3((p.T + R - 1) / R), dim3((p.H / COLS_PER_WARP) * 32), smem, st, p);
  note_launch(1);
  return e != cudaSuccess ? e : cudaGetLastError();
}

template <int MB, bool DH_F32>
cudaError_t launch_bwd(const BwdArgs& p, cudaStream_t st) {
  const size_t smem = rows_smem(p.H, MB);
  const int sz = size_class(p.H);
  auto k = sz == 0 ? adapter_bwd_rows_mma_kernel<MB, 0, DH_F32>
         : sz == 1 ? adapter_bwd_rows_mma_kernel<MB, 1, DH_F32> : adapter_bwd_rows_mma_kernel<MB, 2, DH_F32>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  e = launch_pdl(k, dim3((p.T + R - 1) / R), dim3((p.H / COLS_PER_WARP) * 32), smem, st, p);
  note_launch(1);
  return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace

bool adapter_mma_ok(int H, int m) {
  return H % 128 == 0 && H <= 2048 && (m == 32 || m == 64 || m == 128) &&
         rows_smem(H, m) <= 220 * 1024 && fwd_layout(H, m, 0).bytes <= 220 * 1024;
}

cudaError_t adapter_fwd_mma(const AdapterFwdArgs& a, const void* WdT_b, const void* WuT_b,
                            cudaStream_t st) {
  if (a.dtype != DT_BF16 || !adapter_mma_ok(a.H, a.m)) return cudaErrorNotSupported;
  FwdArgs p;
  p.T = a.T; p.H = a.H; p.m = a.m;
  p.a = reinterpret_cast<const bf16*>(a.a);
  p.WdT = reinterpret_cast<const bf16*>(WdT_b);
  p.WuT = reinterpret_cast<const bf16*>(WuT_b);
  p.z = a.z; p.resid = a.resid; p.gamma = a.gamma; p.beta = a.beta; p.eps = a.eps;
  p.y = reinterpret_cast<bf16*>(a.y); p.x_out = a.x_out;
  p.xhat = reinterpret_cast<bf16*>(a.xhat); p.rstd = a.rstd;
  if (a.no_norm && (a.decoder || a.resid)) return cudaErrorNotSupported;
  const int mode = a.no_norm ? FWD_NONE : a.decoder ? FWD_RMS : FWD_LN;
#define RA_FWD_MODES(MB)                                                          \
  return mode == FWD_NONE ? launch_fwd<MB, FWD_NONE>(p, st)                       \
       : mode == FWD_RMS  ? launch_fwd<MB, FWD_RMS>(p, st) : launch_fwd<MB, FWD_LN>(p, st)
  switch (a.m) {
    case 32: RA_FWD_MODES(32);
    case 64: RA_FWD_MODES(64);
    case 128: RA_FWD_MODES(128);
  }
#undef RA_FWD_MODES
  return cudaErrorNotSupported;
}

cudaError_t adapter_bwd_mma(const AdapterBwdArgs& a, const void* Wu_b, const void* Wd_b,
                            cudaStream_t st) {
  if (a.dtype != DT_BF16 || !adapter_mma_ok(a.H, a.m)) return cudaErrorNotSupported;
  BwdArgs p;
  p.T = a.T; p.H = a.H; p.m = a.m; p.g = a.g; p.z = a.z;
  p.Wu = reinterpret_cast<const bf16*>(Wu_b);
  p.Wd = reinterpret_cast<const bf16*>(Wd_b);
  p.dz = a.dz; p.dh = a.dh;
  const bool f32 = a.dh && a.dh_dtype == DT_F32;
  cudaError_t e = cudaErrorNotSupported;
  if (a.m == 32) e = f32 ? launch_bwd<32, true>(p, st) : launch_bwd<32, false>(p, st);
  else if (a.m == 64) e = f32 ? launch_bwd<64, true>(p, st) : launch_bwd<64, false>(p, st);
  else if (a.m == 128) e = f32 ? launch_bwd<128, true>(p, st) : launch_bwd<128, false>(p, st);
  if (e != cudaSuccess) return e;
  // weight-gradient partials on the tensor cores, then the fixed-order sum
  DwArgs d;
  d.T = a.T; d.H = a.H; d.m = a.m; d.g = a.g; d.h = reinterpret_cast<const bf16*>(a.h);
  d.s = reinterpret_cast<const bf16*>(a.dz);
  d.dz = d.s + (size_t)a.T * a.m;
  d.partials = a.partials;
  const int nchunk = adapter_dw_chunks(a.T, a.H);
  d.chunk = (a.T + nchunk - 1) / nchunk;
  dim3 grid(a.H / DWC, nchunk);
  if (a.m == 32) e = launch_pdl(adapter_dw_mma_kernel<32>, grid, dim3(256), (size_t)0, st, d);
  else if (a.m == 64) e = launch_pdl(adapter_dw_mma_kernel<64>, grid, dim3(256), (size_t)0, st, d);
  else e = launch_pdl(adapter_dw_mma_kernel<128>, grid, dim3(256), (size_t)0, st, d);
  note_launch(1);
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  return adapter_dw_reduce(a.partials, nchunk, a.H, a.m, a.dWd, a.dWu, st);
}

}  // namespace ra
