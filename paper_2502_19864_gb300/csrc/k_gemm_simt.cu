// k_gemm_simt.cu -- CUDA-core GEMM with the step's fused epilogues.
//
// C[M, N] = A[M, K] B[N, K]^T, fp32 accumulation.  This is the path of the fp32 model
// (tcgen05 has no fp32-in/fp32-accurate mode: tf32 keeps 10 mantissa bits, which cannot
// meet a 1e-4 relative bar) and of shapes the tensor-core kernel does not take.
#include "common.cuh"
#include "kernels.h"

namespace ra {
namespace {

constexpr int BM = 64, BN = 64, BK = 16, NT = 256;

template <typename T>
__device__ __forceinline__ float ld(const void* p, int64_t i) {
  return to_f(reinterpret_cast<const T*>(p)[i]);
}
__device__ __forceinline__ float ld_dt(const void* p, int dt, int64_t i) {
  return dt == DT_BF16 ? ld<bf16>(p, i) : ld<float>(p, i);
}
__device__ __forceinline__ void st_dt(void* p, int dt, int64_t i, float v) {
  if (dt == DT_BF16) reinterpret_cast<bf16*>(p)[i] = __float2bfloat16_rn(v);
  else reinterpret_cast<float*>(p)[i] = v;
}

// packed gate/up layout: 64-column blocks alternate gate, up
__device__ __forceinline__ int64_t gate_col(int j) { return (int64_t)(j >> 6) * 128 + (j & 63); }

__device__ __forceinline__ void epilogue(const GemmArgs& g, int m, int n, float acc) {
  switch (g.epi) {
    case EPI_STORE:
    case EPI_SWIGLU: {
      if (g.bias) acc += g.bias[n];
      st_dt(g.C, g.c_dtype, (int64_t)m * g.ldc + n, acc);
    } break;
    case EPI_BIAS_GELU: {
      float u = acc + (g.bias ? g.bias[n] : 0.f);
      if (g.C) st_dt(g.C, g.c_dtype, (int64_t)m * g.ldc + n, u);
      st_dt(g.C2, g.c2_dtype, (int64_t)m * g.ldc2 + n, gelu_f(u));
    } break;
    case EPI_BIAS_GELU_G: {
      float u = acc + (g.bias ? g.bias[n] : 0.f);
      if (g.C) st_dt(g.C, g.c_dtype, (int64_t)m * g.ldc + n, gelu_grad_f(u));
      st_dt(g.C2, g.c2_dtype, (int64_t)m * g.ldc2 + n, gelu_f(u));
    } break;
    case EPI_MUL: {
      float f = ld_dt(g.aux, g.aux_dtype, (int64_t)m * g.ldaux + n);
      st_dt(g.C, g.c_dtype, (int64_t)m * g.ldc + n, acc * f);
    } break;
    case EPI_RESID: {
      float r = ld_dt(g.aux, g.aux_dtype, (int64_t)m * g.ldaux + n);
      st_dt(g.C, g.c_dtype, (int64_t)m * g.ldc + n, acc + r);
    } break;
    case EPI_DSWIGLU: {
      int64_t gc = gate_col(n), uc = gc + 64;
      float gt = ld_dt(g.aux, g.aux_dtype, (int64_t)m * g.ldaux + gc);
      float up = ld_dt(g.aux, g.aux_dtype, (int64_t)m * g.ldaux + uc);
      st_dt(g.C, g.c_dtype, (int64_t)m * g.ldc + gc, acc * up * silu_grad_f(gt));
      st_dt(g.C, g.c_dtype, (int64_t)m * g.ldc + uc, acc * silu_f(gt));
    } break;
  }
}

template <typename TI>
__global__ void __launch_bounds__(NT) gemm_simt_kernel(GemmArgs g) {
  __shared__ float As[BK][BM + 4];
  __shared__ float Bs[BK][BN + 4];
  const int tid = threadIdx.x;
  const int tx = tid & 15, ty = tid >> 4;
  const int m0 = blockIdx.y * BM, n0 = blockIdx.x * BN;
  const TI* A = reinterpret_cast<const TI*>(g.A);
  const TI* B = reinterpret_cast<const TI*>(g.B);
  float acc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;

  for (int k0 = 0; k0 < g.K; k0 += BK) {
    // 64 x 16 tiles: 1024 elements, 4 per thread; k fastest for coalescing
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      int e = tid + r * NT;
      int row = e >> 4, kk = e & 15;
      int gm = m0 + row, gk = k0 + kk;
      As[kk][row] = (gm < g.M && gk < g.K) ? to_f(A[(int64_t)gm * g.lda + gk]) : 0.f;
      if (g.b_kn) {  // B stored [K, N]: n fastest for coalescing
        int n = e & 63, k = e >> 6, gn = n0 + n, gk2 = k0 + k;
        Bs[k][n] = (gn < g.N && gk2 < g.K) ? to_f(B[(int64_t)gk2 * g.ldb + gn]) : 0.f;
      } else {
        int gn = n0 + row;
        Bs[kk][row] = (gn < g.N && gk < g.K) ? to_f(B[(int64_t)gn * g.ldb + gk]) : 0.f;
      }
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < BK; ++kk) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = As[kk][ty + 16 * i];
#pragma unroll
      for (int j = 0; j < 4; ++j) b[j] = Bs[kk][tx + 16 * j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    int m = m0 + ty + 16 * i;
    if (m >= g.M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      int n = n0 + tx + 16 * j;
      if (n < g.N) epilogue(g, m, n, acc[i][j]);
    }
  }
}

// h[m, j] = silu(gate) * up from the packed [gate|up] matrix
__global__ void swiglu_kernel(const void* gu, int ld_gu, int gu_dtype, void* h, int ld_h,
                              int h_dtype, int M, int F) {
  int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (int64_t)M * F) return;
  int m = (int)(idx / F), j = (int)(idx % F);
  int64_t gc = gate_col(j);
  float gt = ld_dt(gu, gu_dtype, (int64_t)m * ld_gu + gc);
  float up = ld_dt(gu, gu_dtype, (int64_t)m * ld_gu + gc + 64);
  st_dt(h, h_dtype, (int64_t)m * ld_h + j, silu_f(gt) * up);
}

}  // namespace

cudaError_t gemm_simt(const GemmArgs& g, cudaStream_t st) {
  if (g.M <= 0 || g.N <= 0) return cudaSuccess;
  dim3 grid((g.N + BN - 1) / BN, (g.M + BM - 1) / BM);
  if (g.in_dtype == DT_BF16) gemm_simt_kernel<bf16><<<grid, NT, 0, st>>>(g);
  else gemm_simt_kernel<float><<<grid, NT, 0, st>>>(g);
  note_launch(1);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess || g.epi != EPI_SWIGLU) return e;
  int F = g.N / 2;
  int64_t n = (int64_t)g.M * F;
  swiglu_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(g.C, g.ldc, g.c_dtype, g.C2,
                                                             g.ldc2, g.c2_dtype, g.M, F);
  note_launch(1);
  return cudaGetLastError();
}

cudaError_t gemm(const GemmArgs& g, cudaStream_t st) {
  if (g.in_dtype == DT_BF16 && tc_available()) {
    cudaError_t e = gemm_tc(g, st);
    if (e != cudaErrorNotSupported) return e;
  }
  return gemm_simt(g, st);
}

}  // namespace ra
