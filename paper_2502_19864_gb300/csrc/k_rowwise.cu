// k_rowwise.cu -- row-wise fused kernels of the step: adapters (Eq. 1) fused with the
// residual add and the block's normalisation, the adapter backward with its in-kernel
// deterministic weight-gradient reduction, LayerNorm / RMSNorm, the heads and their
// cross-entropy, and Adam.
#include "common.cuh"
#include "kernels.h"

namespace ra {
namespace {

template <typename T>
__device__ __forceinline__ float ldf(const void* p, int64_t i) {
  return to_f(reinterpret_cast<const T*>(p)[i]);
}
template <typename T>
__device__ __forceinline__ void stf(void* p, int64_t i, float v) {
  reinterpret_cast<T*>(p)[i] = from_f<T>(v);
}

constexpr int WARPS = 8;
constexpr int RPW = 2;             // rows per warp in the adapter row kernels
constexpr int ROWS = WARPS * RPW;  // rows per CTA
constexpr int MAXM = 128;          // adapter bottleneck upper bound
constexpr int MC = MAXM / 32;      // bottleneck columns per lane

// ---------------------------------------------------------------------------------------
// Adapter forward (Eq. 1) + residual + norm.  Warp w owns rows (blockIdx*ROWS + w*RPW + r).
// smem: rows [ROWS][H] f32 (adapter input, then the pre-norm sum), s [ROWS][m] f32.
// ---------------------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(WARPS * 32) adapter_fwd_kernel(AdapterFwdArgs a) {
  extern __shared__ float sm[];
  const int H = a.H, m = a.m;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float* rows = sm + (size_t)warp * RPW * H;
  float* sv = sm + (size_t)ROWS * H + warp * RPW * MAXM;
  const int t0 = blockIdx.x * ROWS + warp * RPW;

  for (int r = 0; r < RPW; ++r) {
    int t = t0 + r;
    for (int i = lane; i < H; i += 32) rows[r * H + i] = t < a.T ? ldf<T>(a.a, (int64_t)t * H + i) : 0.f;
  }
  __syncwarp();
  // z = a W_down  (lanes over bottleneck columns j = lane + 32c)
  float z[RPW][MC];
#pragma unroll
  for (int r = 0; r < RPW; ++r)
#pragma unroll
    for (int c = 0; c < MC; ++c) z[r][c] = 0.f;
  for (int i = 0; i < H; ++i) {
    float w[MC];
#pragma unroll
    for (int c = 0; c < MC; ++c) {
      int j = lane + 32 * c;
      w[c] = j < m ? a.Wd[(int64_t)i * m + j] : 0.f;
    }
#pragma unroll
    for (int r = 0; r < RPW; ++r) {
      float x = rows[r * H + i];
#pragma unroll
      for (int c = 0; c < MC; ++c) z[r][c] = fmaf(x, w[c], z[r][c]);
    }
  }
#pragma unroll
  for (int r = 0; r < RPW; ++r) {
    int t = t0 + r;
#pragma unroll
    for (int c = 0; c < MC; ++c) {
      int j = lane + 32 * c;
      if (j < m) {
        sv[r * MAXM + j] = gelu_f(z[r][c]);
        if (a.z && t < a.T) a.z[(int64_t)t * m + j] = z[r][c];
      }
    }
  }
  __syncwarp();
  // out = a + GELU(z) W_up, in chunks of 256 columns (lanes over i = i0 + lane + 32cc)
  for (int i0 = 0; i0 < H; i0 += 256) {
    float acc[RPW][8];
#pragma unroll
    for (int r = 0; r < RPW; ++r)
#pragma unroll
      for (int cc = 0; cc < 8; ++cc) acc[r][cc] = 0.f;
    for (int j = 0; j < m; ++j) {
      float w[8];
#pragma unroll
      for (int cc = 0; cc < 8; ++cc) {
        int i = i0 + lane + 32 * cc;
        w[cc] = i < H ? a.Wu[(int64_t)j * H + i] : 0.f;
      }
#pragma unroll
      for (int r = 0; r < RPW; ++r) {
        float s = sv[r * MAXM + j];
#pragma unroll
        for (int cc = 0; cc < 8; ++cc) acc[r][cc] = fmaf(s, w[cc], acc[r][cc]);
      }
    }
#pragma unroll
    for (int r = 0; r < RPW; ++r) {
      int t = t0 + r;
#pragma unroll
      for (int cc = 0; cc < 8; ++cc) {
        int i = i0 + lane + 32 * cc;
        if (i < H) {
          float res = 0.f;
          if (t < a.T && a.resid)
            res = a.decoder ? reinterpret_cast<const float*>(a.resid)[(int64_t)t * H + i]
                            : ldf<T>(a.resid, (int64_t)t * H + i);
          rows[r * H + i] = res + rows[r * H + i] + acc[r][cc];
        }
      }
    }
  }
  __syncwarp();
  // normalisation of the residual sum
  for (int r = 0; r < RPW; ++r) {
    int t = t0 + r;
    if (t >= a.T) break;
    float* v = rows + r * H;
    if (a.no_norm) {
      for (int i = lane; i < H; i += 32) stf<T>(a.y, (int64_t)t * H + i, v[i]);
    } else if (!a.decoder) {
      float s = 0.f;
      for (int i = lane; i < H; i += 32) s += v[i];
      float mu = warp_sum(s) / H;
      float q = 0.f;
      for (int i = lane; i < H; i += 32) { float d = v[i] - mu; q += d * d; }
      float rstd = rsqrtf(warp_sum(q) / H + a.eps);
      for (int i = lane; i < H; i += 32) {
        float xh = (v[i] - mu) * rstd;
        stf<T>(a.y, (int64_t)t * H + i, xh * a.gamma[i] + a.beta[i]);
        if (a.xhat) stf<T>(a.xhat, (int64_t)t * H + i, xh);
      }
      if (a.rstd && lane == 0) a.rstd[t] = rstd;
    } else {
      float q = 0.f;
      for (int i = lane; i < H; i += 32) q += v[i] * v[i];
      float rstd = rsqrtf(warp_sum(q) / H + a.eps);
      for (int i = lane; i < H; i += 32) {
        a.x_out[(int64_t)t * H + i] = v[i];
        stf<T>(a.y, (int64_t)t * H + i, v[i] * rstd * a.gamma[i]);
      }
      if (a.rstd && lane == 0) a.rstd[t] = rstd;
    }
  }
}

// ---------------------------------------------------------------------------------------
// Adapter backward, row part: dz = (g W_up^T) * GELU'(z), dh = g + dz W_down^T
// ---------------------------------------------------------------------------------------
template <typename TO>
__global__ void __launch_bounds__(WARPS * 32) adapter_bwd_rows_kernel(AdapterBwdArgs a) {
  extern __shared__ float sm[];
  const int H = a.H, m = a.m;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float* rows = sm + (size_t)warp * RPW * H;
  float* dzs = sm + (size_t)ROWS * H + warp * RPW * MAXM;
  const int t0 = blockIdx.x * ROWS + warp * RPW;
  for (int r = 0; r < RPW; ++r) {
    int t = t0 + r;
    for (int i = lane; i < H; i += 32) rows[r * H + i] = t < a.T ? a.g[(int64_t)t * H + i] : 0.f;
  }
  __syncwarp();
  float ds[RPW][MC];
#pragma unroll
  for (int r = 0; r < RPW; ++r)
#pragma unroll
    for (int c = 0; c < MC; ++c) ds[r][c] = 0.f;
  for (int i = 0; i < H; ++i) {
    float w[MC];
#pragma unroll
    for (int c = 0; c < MC; ++c) {
      int j = lane + 32 * c;
      w[c] = j < m ? a.WuT[(int64_t)i * m + j] : 0.f;
    }
#pragma unroll
    for (int r = 0; r < RPW; ++r) {
      float x = rows[r * H + i];
#pragma unroll
      for (int c = 0; c < MC; ++c) ds[r][c] = fmaf(x, w[c], ds[r][c]);
    }
  }
#pragma unroll
  for (int r = 0; r < RPW; ++r) {
    int t = t0 + r;
#pragma unroll
    for (int c = 0; c < MC; ++c) {
      int j = lane + 32 * c;
      if (j < m) {
        float dz = 0.f;
        if (t < a.T) {
          dz = ds[r][c] * gelu_grad_f(a.z[(int64_t)t * m + j]);
          a.dz[(int64_t)t * m + j] = dz;
        }
        dzs[r * MAXM + j] = dz;
      }
    }
  }
  __syncwarp();
  if (!a.dh) return;
  for (int i0 = 0; i0 < H; i0 += 256) {
    float acc[RPW][8];
#pragma unroll
    for (int r = 0; r < RPW; ++r)
#pragma unroll
      for (int cc = 0; cc < 8; ++cc) acc[r][cc] = 0.f;
    for (int j = 0; j < m; ++j) {
      float w[8];
#pragma unroll
      for (int cc = 0; cc < 8; ++cc) {
        int i = i0 + lane + 32 * cc;
        w[cc] = i < H ? a.WdT[(int64_t)j * H + i] : 0.f;
      }
#pragma unroll
      for (int r = 0; r < RPW; ++r) {
        float d = dzs[r * MAXM + j];
#pragma unroll
        for (int cc = 0; cc < 8; ++cc) acc[r][cc] = fmaf(d, w[cc], acc[r][cc]);
      }
    }
#pragma unroll
    for (int r = 0; r < RPW; ++r) {
      int t = t0 + r;
      if (t >= a.T) continue;
#pragma unroll
      for (int cc = 0; cc < 8; ++cc) {
        int i = i0 + lane + 32 * cc;
        if (i < H) stf<TO>(a.dh, (int64_t)t * H + i, rows[r * H + i] + acc[r][cc]);
      }
    }
  }
}

// Weight-gradient partials over a chunk of rows:
//   pWu[c][j][i]  = sum_{t in chunk c} GELU(z[t, j]) g[t, i]          (dW_up  = GELU(z)^T g)
//   pWdT[c][j][i] = sum_{t in chunk c} h[t, i] dz[t, j]                (dW_down^T = dz^T h)
// CTA: 64 columns i x all m; thread owns i = tid % 64, j = tid/64 + 4c.
constexpr int DW_COLS = 64, DW_ROWS = 16;
template <typename T>
__global__ void __launch_bounds__(256) adapter_dw_partial_kernel(AdapterBwdArgs a, int chunk) {
  __shared__ float gS[DW_ROWS][DW_COLS], hS[DW_ROWS][DW_COLS];
  __shared__ float sS[DW_ROWS][MAXM], dzS[DW_ROWS][MAXM];
  const int H = a.H, m = a.m;
  const int i0 = blockIdx.x * DW_COLS, c = blockIdx.y;
  const int tid = threadIdx.x, il = tid % DW_COLS, jg = tid / DW_COLS;
  const int tb = c * chunk, te = min(a.T, tb + chunk);
  float aWu[MAXM / 4], aWd[MAXM / 4];
#pragma unroll
  for (int q = 0; q < MAXM / 4; ++q) { aWu[q] = 0.f; aWd[q] = 0.f; }
  for (int t0 = tb; t0 < te; t0 += DW_ROWS) {
    __syncthreads();
    for (int e = tid; e < DW_ROWS * DW_COLS; e += 256) {
      int r = e / DW_COLS, i = e % DW_COLS, t = t0 + r;
      bool in = t < te && i0 + i < H;
      gS[r][i] = in ? a.g[(int64_t)t * H + i0 + i] : 0.f;
      hS[r][i] = in ? ldf<T>(a.h, (int64_t)t * H + i0 + i) : 0.f;
    }
    for (int e = tid; e < DW_ROWS * MAXM; e += 256) {
      int r = e / MAXM, j = e % MAXM, t = t0 + r;
      bool in = t < te && j < m;
      sS[r][j] = in ? gelu_f(a.z[(int64_t)t * m + j]) : 0.f;
      dzS[r][j] = in ? a.dz[(int64_t)t * m + j] : 0.f;
    }
    __syncthreads();
#pragma unroll 4
    for (int r = 0; r < DW_ROWS; ++r) {
      float gv = gS[r][il], hv = hS[r][il];
#pragma unroll
      for (int q = 0; q < MAXM / 4; ++q) {
        int j = jg + 4 * q;
        aWu[q] = fmaf(sS[r][j], gv, aWu[q]);
        aWd[q] = fmaf(dzS[r][j], hv, aWd[q]);
      }
    }
  }
  if (i0 + il >= H) return;
  float* pWu = a.partials + (size_t)c * 2 * H * m;
  float* pWdT = pWu + (size_t)H * m;
#pragma unroll
  for (int q = 0; q < MAXM / 4; ++q) {
    int j = jg + 4 * q;
    if (j < m) {
      pWu[(size_t)j * H + i0 + il] = aWu[q];
      pWdT[(size_t)j * H + i0 + il] = aWd[q];
    }
  }
}

// Fixed-order sum of the partials: dW_up[j][i] and dW_down[i][j].
__global__ void adapter_dw_reduce_kernel(const float* partials, int nchunk, int H, int m,
                                         float* dWd, float* dWu) {
  pdl_wait();
  pdl_trigger();
  int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  int64_t n = (int64_t)H * m;
  if (e >= 2 * n) return;
  bool up = e < n;
  int64_t idx = up ? e : e - n;  // index into [m][H]
  const float* src = partials + (up ? 0 : n) + idx;
  const size_t stride = (size_t)2 * n;
  float s = 0.f;
  int c = 0;
  for (; c + 8 <= nchunk; c += 8) {  // eight loads in flight, summed in chunk order
    float v[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) v[k] = src[(size_t)(c + k) * stride];
#pragma unroll
    for (int k = 0; k < 8; ++k) s += v[k];
  }
  for (; c < nchunk; ++c) s += src[(size_t)c * stride];
  if (up) dWu[idx] = s;
  else {
    int j = (int)(idx / H), i = (int)(idx % H);
    dWd[(int64_t)i * m + j] = s;
  }
}

// Chunk count of the weight-gradient reduction: a pure function of (T, H), so the scratch
// size planned on the host and the grid launched on any device agree, and the reduction
// order (hence the bits of the result) does not depend on the device.
constexpr int kDwTargetCtas = 304;
int dw_chunks(int T, int H) {
  int colblocks = (H + DW_COLS - 1) / DW_COLS;
  int want = (kDwTargetCtas + colblocks - 1) / colblocks;
  int maxc = (T + DW_ROWS - 1) / DW_ROWS;
  return max(1, min(min(want, 64), maxc));
}

// ---------------------------------------------------------------------------------------
// Norms
// ---------------------------------------------------------------------------------------
template <typename T>
__global__ void layernorm_bwd_kernel(const float* dy, const float* dy2, const void* xhat, const float* rstd,
                                     const float* gamma, float* ds, void* ds_act, int Tn, int H) {
  int t = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (t >= Tn) return;
  float s1 = 0.f, s2 = 0.f;
  for (int i = lane; i < H; i += 32) {
    float gy = (dy[(int64_t)t * H + i] + (dy2 ? dy2[(int64_t)t * H + i] : 0.f)) * gamma[i];
    float xh = ldf<T>(xhat, (int64_t)t * H + i);
    s1 += gy;
    s2 += gy * xh;
  }
  s1 = warp_sum(s1) / H;
  s2 = warp_sum(s2) / H;
  float r = rstd[t];
  for (int i = lane; i < H; i += 32) {
    float gy = (dy[(int64_t)t * H + i] + (dy2 ? dy2[(int64_t)t * H + i] : 0.f)) * gamma[i];
    float xh = ldf<T>(xhat, (int64_t)t * H + i);
    const float d = r * (gy - s1 - xh * s2);
    ds[(int64_t)t * H + i] = d;
    if (ds_act) stf<T>(ds_act, (int64_t)t * H + i, d);
  }
}

// LayerNorm of a residual sum: y = LN(x + a) * gamma + beta; xhat and rstd saved when given.
// One warp per row (any H); x, a, y and xhat in the activation type.
template <typename T>
__global__ void add_layernorm_fwd_kernel(const void* x, const void* a, const float* gamma,
                                         const float* beta, float eps, void* y, void* xhat,
                                         float* rstd_out, int Tn, int H) {
  int t = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (t >= Tn) return;
  const int64_t base = (int64_t)t * H;
  float s = 0.f;
  for (int i = lane; i < H; i += 32) s += ldf<T>(x, base + i) + ldf<T>(a, base + i);
  const float mu = warp_sum(s) / H;
  float q = 0.f;
  for (int i = lane; i < H; i += 32) {
    const float d = ldf<T>(x, base + i) + ldf<T>(a, base + i) - mu;
    q += d * d;
  }
  const float r = rsqrtf(warp_sum(q) / H + eps);
  for (int i = lane; i < H; i += 32) {
    const float xh = (ldf<T>(x, base + i) + ldf<T>(a, base + i) - mu) * r;
    stf<T>(y, base + i, xh * gamma[i] + beta[i]);
    if (xhat) stf<T>(xhat, base + i, xh);
  }
  if (rstd_out && lane == 0) rstd_out[t] = r;
}

template <typename TX, typename TN>
__global__ void rmsnorm_fwd_kernel(const void* x, const float* gamma, float eps, void* n,
                                   float* rstd, float* xf, int Tn, int H) {
  int t = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (t >= Tn) return;
  float q = 0.f;
  for (int i = lane; i < H; i += 32) { float v = ldf<TX>(x, (int64_t)t * H + i); q += v * v; }
  float r = rsqrtf(warp_sum(q) / H + eps);
  for (int i = lane; i < H; i += 32) {
    float v = ldf<TX>(x, (int64_t)t * H + i);
    stf<TN>(n, (int64_t)t * H + i, v * r * gamma[i]);
    if (xf) xf[(int64_t)t * H + i] = v;
  }
  if (rstd && lane == 0) rstd[t] = r;
}

__global__ void rmsnorm_bwd_kernel(const float* dy, const float* x, const float* rstd,
                                   const float* gamma, const float* resid, float* dx, int Tn,
                                   int H) {
  int t = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (t >= Tn) return;
  float s = 0.f;
  for (int i = lane; i < H; i += 32) s += dy[(int64_t)t * H + i] * gamma[i] * x[(int64_t)t * H + i];
  s = warp_sum(s) / H;
  float r = rstd[t];
  for (int i = lane; i < H; i += 32) {
    int64_t e = (int64_t)t * H + i;
    float v = r * dy[e] * gamma[i] - x[e] * r * r * r * s;
    dx[e] = (resid ? resid[e] : 0.f) + v;
  }
}

// ---------------------------------------------------------------------------------------
// Row-resident norm kernels for H = 128 V: one warp per row, the row held in registers
// (V float4 per lane, lane-contiguous so a warp access is 512 contiguous bytes), one pass
// over memory.  Same arithmetic as the kernels above, with vector accesses.
// ---------------------------------------------------------------------------------------
template <typename T> __device__ __forceinline__ float4 ld4(const void* p, int64_t i);
template <> __device__ __forceinline__ float4 ld4<float>(const void* p, int64_t i) {
  return *reinterpret_cast<const float4*>(reinterpret_cast<const float*>(p) + i);
}
template <> __device__ __forceinline__ float4 ld4<bf16>(const void* p, int64_t i) {
  const uint2 u = *reinterpret_cast<const uint2*>(reinterpret_cast<const bf16*>(p) + i);
  const float2 a = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.x));
  const float2 b = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.y));
  return make_float4(a.x, a.y, b.x, b.y);
}
template <typename T> __device__ __forceinline__ void st4(void* p, int64_t i, float4 v);
template <> __device__ __forceinline__ void st4<float>(void* p, int64_t i, float4 v) {
  *reinterpret_cast<float4*>(reinterpret_cast<float*>(p) + i) = v;
}
template <> __device__ __forceinline__ void st4<bf16>(void* p, int64_t i, float4 v) {
  __nv_bfloat162 a = __floats2bfloat162_rn(v.x, v.y), b = __floats2bfloat162_rn(v.z, v.w);
  uint2 u;
  u.x = *reinterpret_cast<uint32_t*>(&a);
  u.y = *reinterpret_cast<uint32_t*>(&b);
  *reinterpret_cast<uint2*>(reinterpret_cast<bf16*>(p) + i) = u;
}

template <typename TX, int V>
__global__ void __launch_bounds__(256) layernorm_bwd_vec_kernel(const float* dy, const float* dy2,
    const void* xhat, const float* rstd, const float* gamma, float* ds, void* ds_act, int Tn, int H) {
  pdl_wait();
  pdl_trigger();
  const int row = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (row >= Tn) return;
  const int64_t base = (int64_t)row * H;
  float4 g[V], x[V];
  float s1 = 0.f, s2 = 0.f;
#pragma unroll
  for (int v = 0; v < V; ++v) {
    const int c = (v * 32 + lane) * 4;
    float4 d = ld4<float>(dy, base + c);
    if (dy2) {
      const float4 d2 = ld4<float>(dy2, base + c);
      d = make_float4(d.x + d2.x, d.y + d2.y, d.z + d2.z, d.w + d2.w);
    }
    const float4 gm = ld4<float>(gamma, c);
    g[v] = make_float4(d.x * gm.x, d.y * gm.y, d.z * gm.z, d.w * gm.w);
    x[v] = ld4<TX>(xhat, base + c);
    s1 += g[v].x + g[v].y + g[v].z + g[v].w;
    s2 += g[v].x * x[v].x + g[v].y * x[v].y + g[v].z * x[v].z + g[v].w * x[v].w;
  }
  s1 = warp_sum(s1) / H;
  s2 = warp_sum(s2) / H;
  const float r = rstd[row];
#pragma unroll
  for (int v = 0; v < V; ++v) {
    const int c = (v * 32 + lane) * 4;
    const float4 d = make_float4(r * (g[v].x - s1 - x[v].x * s2), r * (g[v].y - s1 - x[v].y * s2),
                                 r * (g[v].z - s1 - x[v].z * s2), r * (g[v].w - s1 - x[v].w * s2));
    st4<float>(ds, base + c, d);
    if (ds_act) st4<TX>(ds_act, base + c, d);
  }
}

// Vector form of add_layernorm_fwd_kernel (H a multiple of 128): a warp holds its row in
// registers, V float4 per lane, 16- or 8-byte accesses.
template <typename T, int V>
__global__ void __launch_bounds__(256) add_layernorm_fwd_vec_kernel(const void* x, const void* a,
    const float* gamma, const float* beta, float eps, void* y, void* xhat, float* rstd_out, int Tn,
    int H) {
  pdl_wait();
  pdl_trigger();
  const int row = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (row >= Tn) return;
  const int64_t base = (int64_t)row * H;
  float4 v[V];
  float s = 0.f;
#pragma unroll
  for (int k = 0; k < V; ++k) {
    const int c = (k * 32 + lane) * 4;
    const float4 xa = ld4<T>(x, base + c), aa = ld4<T>(a, base + c);
    v[k] = make_float4(xa.x + aa.x, xa.y + aa.y, xa.z + aa.z, xa.w + aa.w);
    s += v[k].x + v[k].y + v[k].z + v[k].w;
  }
  const float mu = warp_sum(s) / H;
  float q = 0.f;
#pragma unroll
  for (int k = 0; k < V; ++k) {
    const float d0 = v[k].x - mu, d1 = v[k].y - mu, d2 = v[k].z - mu, d3 = v[k].w - mu;
    q += d0 * d0 + d1 * d1 + d2 * d2 + d3 * d3;
  }
  const float r = rsqrtf(warp_sum(q) / H + eps);
#pragma unroll
  for (int k = 0; k < V; ++k) {
    const int c = (k * 32 + lane) * 4;
    const float4 gm = ld4<float>(gamma, c), bt = ld4<float>(beta, c);
    const float4 xh = make_float4((v[k].x - mu) * r, (v[k].y - mu) * r, (v[k].z - mu) * r, (v[k].w - mu) * r);
    st4<T>(y, base + c, make_float4(xh.x * gm.x + bt.x, xh.y * gm.y + bt.y, xh.z * gm.z + bt.z, xh.w * gm.w + bt.w));
    if (xhat) st4<T>(xhat, base + c, xh);
  }
  if (rstd_out && lane == 0) rstd_out[row] = r;
}

template <typename TX, typename TN, int V>
__global__ void __launch_bounds__(256) rmsnorm_fwd_vec_kernel(const void* x, const float* gamma, float eps,
    void* n, float* rstd, float* xf, int Tn, int H) {
  pdl_wait();
  pdl_trigger();
  const int row = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (row >= Tn) return;
  const int64_t base = (int64_t)row * H;
  float4 a[V];
  float q = 0.f;
#pragma unroll
  for (int v = 0; v < V; ++v) {
    a[v] = ld4<TX>(x, base + (v * 32 + lane) * 4);
    q += a[v].x * a[v].x + a[v].y * a[v].y + a[v].z * a[v].z + a[v].w * a[v].w;
  }
  const float r = rsqrtf(warp_sum(q) / H + eps);
#pragma unroll
  for (int v = 0; v < V; ++v) {
    const int c = (v * 32 + lane) * 4;
    const float4 gm = ld4<float>(gamma, c);
    st4<TN>(n, base + c, make_float4(a[v].x * r * gm.x, a[v].y * r * gm.y, a[v].z * r * gm.z, a[v].w * r * gm.w));
    if (xf) st4<float>(xf, base + c, a[v]);
  }
  if (rstd && lane == 0) rstd[row] = r;
}

template <int V>
__global__ void __launch_bounds__(256) rmsnorm_bwd_vec_kernel(const float* dy, const float* x, const float* rstd,
    const float* gamma, const float* resid, float* dx, int Tn, int H) {
  pdl_wait();
  pdl_trigger();
  const int row = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (row >= Tn) return;
  const int64_t base = (int64_t)row * H;
  float4 g[V], a[V];
  float s = 0.f;
#pragma unroll
  for (int v = 0; v < V; ++v) {
    const int c = (v * 32 + lane) * 4;
    const float4 d = ld4<float>(dy, base + c), gm = ld4<float>(gamma, c);
    g[v] = make_float4(d.x * gm.x, d.y * gm.y, d.z * gm.z, d.w * gm.w);
    a[v] = ld4<float>(x, base + c);
    s += g[v].x * a[v].x + g[v].y * a[v].y + g[v].z * a[v].z + g[v].w * a[v].w;
  }
  s = warp_sum(s) / H;
  const float r = rstd[row], k = r * r * r * s;
#pragma unroll
  for (int v = 0; v < V; ++v) {
    const int c = (v * 32 + lane) * 4;
    const float4 q = resid ? ld4<float>(resid, base + c) : make_float4(0.f, 0.f, 0.f, 0.f);
    st4<float>(dx, base + c, make_float4(q.x + r * g[v].x - a[v].x * k, q.y + r * g[v].y - a[v].y * k,
                                         q.z + r * g[v].z - a[v].z * k, q.w + r * g[v].w - a[v].w * k));
  }
}

// V for the row-resident kernels (0: use the scalar kernels)
inline int row_vec(int H) {
  if (H % 128) return 0;
  const int v = H / 128;
  return (v == 1 || v == 2 || v == 4 || v == 6 || v == 8 || v == 16) ? v : 0;
}
#define RA_VEC_SWITCH(V, CALL)                 \
  switch (V) {                                 \
    case 1: { constexpr int VV = 1; CALL; } break;  \
    case 2: { constexpr int VV = 2; CALL; } break;  \
    case 4: { constexpr int VV = 4; CALL; } break;  \
    case 6: { constexpr int VV = 6; CALL; } break;  \
    case 8: { constexpr int VV = 8; CALL; } break;  \
    case 16: { constexpr int VV = 16; CALL; } break; \
  }

// ---------------------------------------------------------------------------------------
// Heads
// ---------------------------------------------------------------------------------------
constexpr int MAXC = 32, MAXB = 256;
constexpr int HEAD_FWD_THREADS = 512, HEAD_BWD_THREADS = 128;
// forward: logits = y[b, 0, :] Wh^T + bh, mean CE, dlogits = (softmax - onehot) / B.
// One warp per batch row computes all C logits of the row at once, with eight loads of the
// CLS row in flight per lane; then one thread per row takes the softmax.  CM >= C is the
// number of class accumulators held in registers (2, 8 or MAXC).
template <typename T, int CM>
__global__ void __launch_bounds__(HEAD_FWD_THREADS) encoder_head_fwd_kernel(const void* y, const float* Wh,
    const float* bh, const int32_t* labels, int B, int S, int H, int C, float* loss,
    float* logits_out, float* dlogits, unsigned* err) {
  __shared__ float lg[MAXB * MAXC];
  __shared__ float red[MAXB];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  for (int b = warp; b < B; b += nw) {
    const int64_t row = (int64_t)b * S * H;
    float acc[CM];
#pragma unroll
    for (int c = 0; c < CM; ++c) acc[c] = 0.f;
    // bf16 rows: 8 columns per lane and load (16 bytes), so a row takes H / 256 round trips
    int i0 = 0;
    if (sizeof(T) == 2 && H % 256 == 0 && ((row * 2) & 15) == 0 &&
        ((reinterpret_cast<uintptr_t>(y) | reinterpret_cast<uintptr_t>(Wh)) & 15) == 0) {
      for (int i = 8 * lane; i < H; i += 256) {
        const uint4 w = *reinterpret_cast<const uint4*>(reinterpret_cast<const T*>(y) + row + i);
        const uint32_t u[4] = {w.x, w.y, w.z, w.w};
        float x[8];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u[q]));
          x[2 * q] = f.x;
          x[2 * q + 1] = f.y;
        }
#pragma unroll
        for (int c = 0; c < CM; ++c)
          if (c < C) {
            const float4 a0 = __ldg(reinterpret_cast<const float4*>(Wh + (int64_t)c * H + i));
            const float4 a1 = __ldg(reinterpret_cast<const float4*>(Wh + (int64_t)c * H + i + 4));
            acc[c] += x[0] * a0.x + x[1] * a0.y + x[2] * a0.z + x[3] * a0.w + x[4] * a1.x + x[5] * a1.y +
                      x[6] * a1.z + x[7] * a1.w;
          }
      }
      i0 = H;
    }
#pragma unroll 8
    for (int i = i0 + lane; i < H; i += 32) {
      const float x = ldf<T>(y, row + i);
#pragma unroll
      for (int c = 0; c < CM; ++c)
        if (c < C) acc[c] += x * __ldg(Wh + (int64_t)c * H + i);
    }
#pragma unroll
    for (int c = 0; c < CM; ++c)
      if (c < C) {
        const float s = warp_sum(acc[c]);
        if (lane == 0) lg[b * C + c] = s + bh[c];
      }
  }
  __syncthreads();
  for (int b = threadIdx.x; b < B; b += blockDim.x) {
    float mx = -INFINITY;
    for (int c = 0; c < C; ++c) mx = fmaxf(mx, lg[b * C + c]);
    float se = 0.f;
    for (int c = 0; c < C; ++c) se += expf(lg[b * C + c] - mx);
    float lse = mx + logf(se);
    int lab = labels[b];
    if (lab < 0 || lab >= C) { set_dev_error(err, RA_DEVERR_BOUNDS); lab = 0; }
    red[b] = lse - lg[b * C + lab];
    for (int c = 0; c < C; ++c) {
      if (logits_out) logits_out[b * C + c] = lg[b * C + c];
      float p = expf(lg[b * C + c] - lse);
      dlogits[b * C + c] = (p - (c == lab ? 1.f : 0.f)) / B;
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float s = 0.f;
    for (int b = 0; b < B; ++b) s += red[b];
    *loss = s / B;
  }
}

// backward: dWh = dlogits^T cls, dbh = sum_b dlogits, dy[b, 0, :] = dlogits Wh.  One thread
// per column i; the column's B CLS values are loaded eight at a time, so a thread waits on
// B / 8 round trips instead of C * B.  CM >= C as in the forward.
template <typename T, int CM>
__global__ void __launch_bounds__(HEAD_BWD_THREADS) encoder_head_bwd_kernel(const void* y, const float* Wh,
    const float* dlogits, int B, int S, int H, int C, float* dWh, float* dbh, float* dy) {
  __shared__ float lg[MAXB * MAXC];
  for (int e = threadIdx.x; e < B * C; e += blockDim.x) lg[e] = dlogits[e];
  __syncthreads();
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < H) {
    float w[CM], acc[CM];
#pragma unroll
    for (int c = 0; c < CM; ++c) {
      acc[c] = 0.f;
      w[c] = c < C ? __ldg(Wh + (int64_t)c * H + i) : 0.f;
    }
    for (int b0 = 0; b0 < B; b0 += 8) {
      float x[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) x[k] = b0 + k < B ? ldf<T>(y, (int64_t)(b0 + k) * S * H + i) : 0.f;
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        if (b0 + k < B) {
          const float* l = lg + (b0 + k) * C;
          float s = 0.f;
#pragma unroll
          for (int c = 0; c < CM; ++c)
            if (c < C) {
              acc[c] += l[c] * x[k];
              s += l[c] * w[c];
            }
          dy[(int64_t)(b0 + k) * S * H + i] = s;
        }
      }
    }
    if (dWh) {
#pragma unroll
      for (int c = 0; c < CM; ++c)
        if (c < C) dWh[(int64_t)c * H + i] = acc[c];
    }
  }
  if (dbh && blockIdx.x == 0 && threadIdx.x < C) {
    float s = 0.f;
    for (int b = 0; b < B; ++b) s += lg[b * C + threadIdx.x];
    dbh[threadIdx.x] = s;
  }
}

// ---------------------------------------------------------------------------------------
// Span head: start and end logits at every token, loss = the mean over the batch of
// (CE_start + CE_end) / 2, each a softmax over the S positions of one sequence.
// ---------------------------------------------------------------------------------------
constexpr int SPAN_CHUNKS = 32;   // token chunks of the deterministic dWh reduction
// forward: one CTA per sequence b.  logits [S, 2] of its tokens (a warp per token, both
// logits at once) into shared memory; warp c then takes the softmax over S of column c and
// writes dlogits[t, c] = (p_c(s) - [s == label_c]) / (2 B); row_loss[b] = mean of the two
// cross-entropies.
// Span head logits: a warp per token, z[t] = (y_t . Wh[0] + bh[0], y_t . Wh[1] + bh[1]) into
// zout [T][2] (the dlogits buffer, which the softmax kernel then overwrites in place).
// 16-byte loads of y (8 bf16 or 4 f32 per load, H a multiple of 8).
template <typename T>
__global__ void __launch_bounds__(256) span_head_logits_kernel(const void* y, const float* Wh,
    const float* bh, int Tn, int H, float* zout) {
  pdl_wait();
  pdl_trigger();
  const int64_t t = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (t >= Tn) return;
  constexpr int V = 16 / sizeof(T);  // elements per 16-byte load
  const T* row = reinterpret_cast<const T*>(y) + t * H;
  float a0 = 0.f, a1 = 0.f;
  for (int i = lane * V; i < H; i += 32 * V) {
    const uint4 u = *reinterpret_cast<const uint4*>(row + i);
    float x[V];
    if (V == 8) {
      const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
      for (int k = 0; k < V / 2; ++k) {
        const float2 f = __bfloat1622float2(h2[k]);
        x[2 * k] = f.x;
        x[2 * k + 1] = f.y;
      }
    } else {
      const float* f = reinterpret_cast<const float*>(&u);
#pragma unroll
      for (int k = 0; k < V; ++k) x[k] = f[k];
    }
#pragma unroll
    for (int k = 0; k < V; ++k) {
      a0 = fmaf(x[k], __ldg(Wh + i + k), a0);
      a1 = fmaf(x[k], __ldg(Wh + H + i + k), a1);
    }
  }
  a0 = warp_sum(a0);
  a1 = warp_sum(a1);
  if (lane == 0) *reinterpret_cast<float2*>(zout + 2 * t) = make_float2(a0 + bh[0], a1 + bh[1]);
}

// Span head softmax and cross-entropy, one CTA per sequence: the start (c = 0) and end (c = 1)
// columns take a warp each.  z [T][2] arrives in dlogits and is replaced by the gradient.
__global__ void __launch_bounds__(64) span_head_ce_kernel(const int32_t* labels, int B, int S,
    float* row_loss, float* logits_out, float* dlogits, unsigned* err) {
  pdl_wait();
  pdl_trigger();
  __shared__ float part[2];
  const int b = blockIdx.x, c = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const float* z = dlogits + (int64_t)b * S * 2;
  int lab = labels[2 * b + c];
  if (lab < 0 || lab >= S) {
    if (lane == 0) set_dev_error(err, RA_DEVERR_BOUNDS);
    lab = 0;
  }
  float mx = -INFINITY;
  for (int s = lane; s < S; s += 32) mx = fmaxf(mx, z[2 * s + c]);
  mx = warp_max(mx);
  float se = 0.f;
  for (int s = lane; s < S; s += 32) se += expf(z[2 * s + c] - mx);
  se = warp_sum(se);
  const float lse = mx + logf(se);
  const float zlab = z[2 * lab + c];
  __syncwarp();
  const float inv = 1.f / (2.f * B);
  for (int s = lane; s < S; s += 32) {
    const int64_t t = (int64_t)b * S + s;
    const float zz = dlogits[2 * t + c];
    if (logits_out) logits_out[2 * t + c] = zz;
    dlogits[2 * t + c] = (expf(zz - lse) - (s == lab ? 1.f : 0.f)) * inv;
  }
  if (lane == 0) part[c] = lse - zlab;
  __syncthreads();
  if (threadIdx.x == 0) row_loss[b] = 0.5f * (part[0] + part[1]);
}

// backward, every token's gradient: dy[t, :] = dlogits[t, 0] Wh[0, :] + dlogits[t, 1] Wh[1, :]
// (a warp per token, 16-byte accesses; H % 4 == 0)
__global__ void __launch_bounds__(256) span_head_dy_kernel(const float* Wh, const float* dlogits,
                                                           int Tn, int H, float* dy) {
  const int64_t t = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (t >= Tn) return;
  const float d0 = dlogits[2 * t], d1 = dlogits[2 * t + 1];
  for (int i = 4 * lane; i < H; i += 128) {
    const float4 w0 = __ldg(reinterpret_cast<const float4*>(Wh + i));
    const float4 w1 = __ldg(reinterpret_cast<const float4*>(Wh + H + i));
    *reinterpret_cast<float4*>(dy + t * H + i) =
        make_float4(d0 * w0.x + d1 * w1.x, d0 * w0.y + d1 * w1.y, d0 * w0.z + d1 * w1.z, d0 * w0.w + d1 * w1.w);
  }
}

// backward, head weights: per chunk c of tokens, part[c][j][i] = sum over the chunk's tokens
// (in token order) of dlogits[t, j] y[t, i] (a thread per column i, eight tokens' loads in
// flight), and part_b[c][j] = the chunk's sum of dlogits[t, j]
template <typename T>
__global__ void __launch_bounds__(128) span_head_dw_kernel(const void* y, const float* dlogits,
    int Tn, int H, int chunk, float* part, float* part_b) {
  const int i = blockIdx.x * 128 + threadIdx.x, c = blockIdx.y;
  const int t0 = c * chunk, t1 = min(Tn, t0 + chunk);
  if (i < H) {
    float a0 = 0.f, a1 = 0.f;
    for (int t = t0; t < t1; t += 8) {
      float x[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) x[k] = t + k < t1 ? ldf<T>(y, (int64_t)(t + k) * H + i) : 0.f;
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        if (t + k < t1) {
          a0 += dlogits[2 * (t + k)] * x[k];
          a1 += dlogits[2 * (t + k) + 1] * x[k];
        }
      }
    }
    part[((size_t)c * 2) * H + i] = a0;
    part[((size_t)c * 2 + 1) * H + i] = a1;
  }
  if (blockIdx.x == 0 && threadIdx.x < 2) {
    float sb = 0.f;
    for (int t = t0; t < t1; ++t) sb += dlogits[2 * t + threadIdx.x];
    part_b[2 * c + threadIdx.x] = sb;
  }
}

// fixed-order sum of the chunk partials: dWh [2, H], dbh [2]
__global__ void __launch_bounds__(256) span_head_dw_reduce_kernel(const float* part, const float* part_b,
    int nch, int H, float* dWh, float* dbh) {
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  if (dWh && j < 2 * H) {
    float s = 0.f;
    for (int c = 0; c < nch; ++c) s += part[(size_t)c * 2 * H + j];
    dWh[j] = s;
  }
  if (dbh && blockIdx.x == 0 && threadIdx.x < 2) {
    float s = 0.f;
    for (int c = 0; c < nch; ++c) s += part_b[2 * c + threadIdx.x];
    dbh[threadIdx.x] = s;
  }
}

// one CTA per row: in-place dlogits = (softmax - onehot) / T
template <typename T>
__global__ void __launch_bounds__(256) vocab_ce_kernel(void* logits, int ld,
    const int32_t* labels, int Tn, int V, float* row_loss, float* logits_out, unsigned* err) {
  __shared__ float red[8];
  const int t = blockIdx.x, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  T* row = reinterpret_cast<T*>(logits) + (int64_t)t * ld;
  float mx = -INFINITY;
  for (int j = threadIdx.x; j < V; j += 256) {
    float v = to_f(row[j]);
    mx = fmaxf(mx, v);
    if (logits_out) logits_out[(int64_t)t * V + j] = v;
  }
  mx = warp_max(mx);
  if (lane == 0) red[warp] = mx;
  __syncthreads();
  mx = red[0];
  for (int w = 1; w < 8; ++w) mx = fmaxf(mx, red[w]);
  __syncthreads();
  float se = 0.f;
  // (the special-function exponential: about 2 ulp, against the dozen-odd instructions of
  // expf per logit over a 32000-wide vocabulary)
  for (int j = threadIdx.x; j < V; j += 256) se += __expf(to_f(row[j]) - mx);
  se = warp_sum(se);
  if (lane == 0) red[warp] = se;
  __syncthreads();
  se = 0.f;
  for (int w = 0; w < 8; ++w) se += red[w];
  float lse = mx + logf(se);
  int lab = labels[t];
  if (lab < 0 || lab >= V) {
    if (threadIdx.x == 0) set_dev_error(err, RA_DEVERR_BOUNDS);
    lab = 0;
  }
  float zl = to_f(row[lab]);
  __syncthreads();
  if (threadIdx.x == 0) row_loss[t] = lse - zl;
  float invT = 1.f / Tn;
  for (int j = threadIdx.x; j < V; j += 256) {
    float p = __expf(to_f(row[j]) - lse);
    row[j] = from_f<T>((p - (j == lab ? 1.f : 0.f)) * invT);
  }
}

__global__ void __launch_bounds__(256) mean_kernel(const float* v, int n, float* out) {
  __shared__ float red[256];
  float s = 0.f;
  for (int i = threadIdx.x; i < n; i += 256) s += v[i];
  red[threadIdx.x] = s;
  __syncthreads();
  for (int w = 128; w > 0; w >>= 1) {
    if (threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) *out = red[0] / n;
}

// ---------------------------------------------------------------------------------------
// Adam
// ---------------------------------------------------------------------------------------
// The bias corrections depend only on the segment's step count: they are evaluated once for
// the segments of a block's first and last element instead of per element (powf twice per
// element dominated the kernel's instructions); only a segment shorter than a block, lying
// strictly inside one, falls back to evaluating them per element.
__global__ void adam_kernel(AdamArgs a) {
  __shared__ float corr[2][2];  // [first / second segment of the block][lr / bc1, 1 / sqrt(bc2)]
  __shared__ int segs[2];
  const int64_t base = (int64_t)blockIdx.x * blockDim.x;
  if (threadIdx.x < 2) {
    const int64_t e = threadIdx.x == 0 ? base : min(a.n - 1, base + (int64_t)blockDim.x - 1);
    const int64_t se = e / a.seg_len;
    const int s = (int)(se < a.n_seg - 1 ? se : a.n_seg - 1);
    const float t = (float)(a.steps[s] + 1);
    corr[threadIdx.x][0] = a.lr / (1.f - powf(a.beta1, t));
    corr[threadIdx.x][1] = 1.f / sqrtf(1.f - powf(a.beta2, t));
    segs[threadIdx.x] = s;
  }
  __syncthreads();
  const int64_t i = base + threadIdx.x;
  if (i >= a.n) return;
  const int64_t si = i / a.seg_len;
  const int s = (int)(si < a.n_seg - 1 ? si : a.n_seg - 1);
  float c[2];
  if (s == segs[0] || s == segs[1]) {
    c[0] = corr[s == segs[0] ? 0 : 1][0];
    c[1] = corr[s == segs[0] ? 0 : 1][1];
  } else {  // a segment shorter than the block, lying strictly inside it
    const float t = (float)(a.steps[s] + 1);
    c[0] = a.lr / (1.f - powf(a.beta1, t));
    c[1] = 1.f / sqrtf(1.f - powf(a.beta2, t));
  }
  const float g = a.g[i];
  const float m = a.beta1 * a.m[i] + (1.f - a.beta1) * g;
  const float v = a.beta2 * a.v[i] + (1.f - a.beta2) * g * g;
  a.m[i] = m;
  a.v[i] = v;
  a.p[i] -= c[0] * m / (sqrtf(v) * c[1] + a.eps);
}

__global__ void bump_kernel(int32_t* steps, int n) {
  int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) steps[i] += 1;
}

// ---------------------------------------------------------------------------------------
// utilities
// ---------------------------------------------------------------------------------------
template <typename T>
__global__ void convert_kernel(const float* src, void* dst, int64_t n) {
  int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) stf<T>(dst, i, src[i]);
}

template <typename T>
__global__ void transpose_kernel(const float* src, void* dst, int rows, int cols, int ld_dst) {
  __shared__ float tile[32][33];
  int c0 = blockIdx.x * 32, r0 = blockIdx.y * 32;
  for (int y = threadIdx.y; y < 32; y += 8) {
    int r = r0 + y, c = c0 + threadIdx.x;
    tile[y][threadIdx.x] = (r < rows && c < cols) ? src[(int64_t)r * cols + c] : 0.f;
  }
  __syncthreads();
  for (int y = threadIdx.y; y < 32; y += 8) {
    int c = c0 + y, r = r0 + threadIdx.x;
    if (c < cols && r < rows) stf<T>(dst, (int64_t)c * ld_dst + r, tile[threadIdx.x][y]);
  }
}

// packed gate/up row of source row r of part (0 = gate, 1 = up): 64-row blocks alternate
__device__ __forceinline__ int64_t packed_row(int r, int part) {
  return (int64_t)(r >> 6) * 128 + part * 64 + (r & 63);
}
template <typename T>
__global__ void pack_rows_kernel(const float* src, void* dst, int R, int C, int part, int transposed) {
  int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= (int64_t)R * C) return;
  int r = (int)(e / C), c = (int)(e % C);
  int64_t pr = packed_row(r, part);
  if (transposed) stf<T>(dst, (int64_t)c * (2 * R) + pr, src[e]);
  else stf<T>(dst, pr * C + c, src[e]);
}

// transposed copies of the adapter matrices of layers [l0, l1): for each layer the four
// matrices WdA [H,m], WuA [m,H], WdF [H,m], WuF [m,H] (contiguous, 4Hm per layer) go to
// WdT [m,H], WuT [H,m], ... at the same offsets of PT.
// Position of element k of a row inside the fragment-major order of the bf16 adapter shadows:
// within each 32-wide block, the values k = 8q + 2t + b (q, b in {0..3}, {0, 1}) that thread
// t of an mma.sync needs for two k16 steps are stored together at 8t + 2q + b.
__device__ __forceinline__ int frag_pos(int k) {
  const int w = k & 31;
  return (k & ~31) + ((w & 7) >> 1) * 8 + (w >> 3) * 2 + (w & 1);
}
// Offset of element (n, k) of a bf16 [R, C] matrix in the tiled fragment layout the
// tensor-core adapter kernels read: 8-row x 32-column blocks of 256 contiguous elements,
// ordered by row block then column block; inside a block, row n & 7 holds its 32 columns in
// the m16n8k16 B-fragment order (frag_pos), so the 32 lanes of a warp load the fragments of
// one n8 tile and two k16 steps as 512 contiguous bytes.
__device__ __forceinline__ int64_t tfrag_off(int n, int k, int C) {
  return ((int64_t)(n >> 3) * (C >> 5) + (k >> 5)) * 256 + (n & 7) * 32 + frag_pos(k & 31);
}

// P (f32 masters) -> PT (f32, transposed) and, for bf16 models, the shadows PB (the master's
// layout [rows, cols]) and PTB (transposed [cols, rows]) in the tiled fragment layout; when
// H or m is not a multiple of 32 (no tensor-core kernel reads them then) they are plain
// row-major copies.
// One block per 32 x 32 tile of one matrix: the tile is read row-major (coalesced, and PB's
// fragment offsets of a 32-column run stay inside one 64-byte span), staged in shared memory,
// and written transposed with the same coalescing for PT and PTB.
__global__ void __launch_bounds__(256) adapter_transpose_kernel(const float* P, float* PT, bf16* PB,
                                                                bf16* PTB, int H, int m) {
  __shared__ float tile[32][33];
  const int layer = blockIdx.z >> 2, mat = blockIdx.z & 3;
  const int64_t base = (int64_t)layer * 4 * H * m + (int64_t)mat * H * m;
  const int rows = (mat & 1) ? m : H, cols = (mat & 1) ? H : m;
  const int tiles_c = (cols + 31) >> 5;
  const int r0 = (int)(blockIdx.x / tiles_c) * 32, c0 = (int)(blockIdx.x % tiles_c) * 32;
  const bool tiled = (H % 32 == 0) && (m % 32 == 0);
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  for (int j = ty; j < 32; j += 8) {
    const int r = r0 + j, c = c0 + tx;
    if (r < rows && c < cols) {
      const int64_t e = (int64_t)r * cols + c;
      const float v = P[base + e];
      tile[j][tx] = v;
      if (PB) PB[base + (tiled ? tfrag_off(r, c, cols) : e)] = __float2bfloat16_rn(v);
    }
  }
  __syncthreads();
  for (int j = ty; j < 32; j += 8) {
    const int c = c0 + j, r = r0 + tx;
    if (r < rows && c < cols) {
      const float v = tile[tx][j];
      const int64_t t = (int64_t)c * rows + r;
      PT[base + t] = v;
      if (PTB) PTB[base + (tiled ? tfrag_off(c, r, rows) : t)] = __float2bfloat16_rn(v);
    }
  }
}

// Adam on the adapter matrices (Algorithm 1's adapter update, the same arithmetic as
// adam_kernel) fused with the refresh of their transposed and bf16 copies: one block per
// 32 x 32 tile of one matrix updates the tile's masters in place, then writes PB from the new
// values and stages them in shared memory for PT and PTB, so P is read once per update
// instead of twice. Every element of a layer shares the layer's step count, hence one bias
// correction per block.
__global__ void __launch_bounds__(256) adam_adapter_kernel(AdamArgs a, float* PT, bf16* PB, bf16* PTB,
                                                           int H, int m) {
  __shared__ float tile[32][33];
  const int layer = blockIdx.z >> 2, mat = blockIdx.z & 3;
  const int64_t base = (int64_t)layer * 4 * H * m + (int64_t)mat * H * m;
  const int rows = (mat & 1) ? m : H, cols = (mat & 1) ? H : m;
  const int tiles_c = (cols + 31) >> 5;
  const int r0 = (int)(blockIdx.x / tiles_c) * 32, c0 = (int)(blockIdx.x % tiles_c) * 32;
  const bool tiled = (H % 32 == 0) && (m % 32 == 0);
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  const float t = (float)(a.steps[layer] + 1);
  const float c_lr = a.lr / (1.f - powf(a.beta1, t)), c_v = 1.f / sqrtf(1.f - powf(a.beta2, t));
  for (int j = ty; j < 32; j += 8) {
    const int r = r0 + j, c = c0 + tx;
    if (r < rows && c < cols) {
      const int64_t e = (int64_t)r * cols + c, i = base + e;
      const float g = a.g[i];
      const float mo = a.beta1 * a.m[i] + (1.f - a.beta1) * g;
      const float vo = a.beta2 * a.v[i] + (1.f - a.beta2) * g * g;
      a.m[i] = mo;
      a.v[i] = vo;
      const float v = a.p[i] - c_lr * mo / (sqrtf(vo) * c_v + a.eps);
      a.p[i] = v;
      tile[j][tx] = v;
      if (PB) PB[base + (tiled ? tfrag_off(r, c, cols) : e)] = __float2bfloat16_rn(v);
    }
  }
  __syncthreads();
  for (int j = ty; j < 32; j += 8) {
    const int c = c0 + j, r = r0 + tx;
    if (r < rows && c < cols) {
      const float v = tile[tx][j];
      const int64_t tt = (int64_t)c * rows + r;
      PT[base + tt] = v;
      if (PTB) PTB[base + (tiled ? tfrag_off(c, r, rows) : tt)] = __float2bfloat16_rn(v);
    }
  }
}

__global__ void activation_kernel(int which, const float* x, float* y, int64_t n) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const float v = x[i];
  y[i] = which == 0 ? gelu_f(v) : which == 1 ? gelu_grad_f(v) : which == 2 ? silu_f(v) : silu_grad_f(v);
}

__global__ void fill_kernel(float* dst, float v, int64_t n) {
  int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) dst[i] = v;
}

inline unsigned blocks_for(int64_t n, int per) { return (unsigned)((n + per - 1) / per); }

}  // namespace

// =========================================================================================
cudaError_t adapter_fwd(const AdapterFwdArgs& a, cudaStream_t st) {
  if (a.m > MAXM || a.m <= 0) return cudaErrorInvalidValue;
  if (a.dtype == DT_BF16 && a.WdT_b && a.WuT_b && adapter_mma_ok(a.H, a.m))
    return adapter_fwd_mma(a, a.WdT_b, a.WuT_b, st);
  size_t smem = ((size_t)ROWS * a.H + ROWS * MAXM) * sizeof(float);
  unsigned grid = blocks_for(a.T, ROWS);
  if (a.dtype == DT_BF16) {
    cudaFuncSetAttribute(adapter_fwd_kernel<bf16>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    adapter_fwd_kernel<bf16><<<grid, WARPS * 32, smem, st>>>(a);
  } else {
    cudaFuncSetAttribute(adapter_fwd_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    adapter_fwd_kernel<float><<<grid, WARPS * 32, smem, st>>>(a);
  }
  note_launch(1);
  return cudaGetLastError();
}

size_t adapter_bwd_partials_floats(int T, int H, int m) {
  return (size_t)dw_chunks(T, H) * 2 * H * m;
}

int adapter_dw_chunks(int T, int H) { return dw_chunks(T, H); }

cudaError_t adapter_dw_reduce(const float* partials, int nchunk, int H, int m, float* dWd,
                              float* dWu, cudaStream_t st) {
  int64_t n = 2LL * H * m;
  (void)launch_pdl(adapter_dw_reduce_kernel, dim3(blocks_for(n, 256)), dim3(256), (size_t)0, st, partials, nchunk, H, m, dWd, dWu);
  note_launch(1);
  return cudaGetLastError();
}

cudaError_t adapter_bwd(const AdapterBwdArgs& a, cudaStream_t st) {
  if (a.m > MAXM || a.m <= 0) return cudaErrorInvalidValue;
  // the tensor-core kernels write dh as bf16 or f32, so whether (and how) dh is wanted
  // never changes which kernels compute dz and dW
  if (a.dtype == DT_BF16 && a.Wu_b && a.Wd_b && adapter_mma_ok(a.H, a.m))
    return adapter_bwd_mma(a, a.Wu_b, a.Wd_b, st);
  size_t smem = ((size_t)ROWS * a.H + ROWS * MAXM) * sizeof(float);
  unsigned grid = blocks_for(a.T, ROWS);
  if (a.dh_dtype == DT_BF16) {
    cudaFuncSetAttribute(adapter_bwd_rows_kernel<bf16>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    adapter_bwd_rows_kernel<bf16><<<grid, WARPS * 32, smem, st>>>(a);
  } else {
    cudaFuncSetAttribute(adapter_bwd_rows_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    adapter_bwd_rows_kernel<float><<<grid, WARPS * 32, smem, st>>>(a);
  }
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  int nchunk = dw_chunks(a.T, a.H);
  int chunk = (a.T + nchunk - 1) / nchunk;
  dim3 g2((a.H + DW_COLS - 1) / DW_COLS, nchunk);
  if (a.dtype == DT_BF16) adapter_dw_partial_kernel<bf16><<<g2, 256, 0, st>>>(a, chunk);
  else adapter_dw_partial_kernel<float><<<g2, 256, 0, st>>>(a, chunk);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  int64_t n = 2LL * a.H * a.m;
  (void)launch_pdl(adapter_dw_reduce_kernel, dim3(blocks_for(n, 256)), dim3(256), (size_t)0, st, a.partials, nchunk, a.H, a.m, a.dWd, a.dWu);
  note_launch(3);
  return cudaGetLastError();
}

cudaError_t layernorm_bwd(const float* dy, const float* dy2, const void* xhat, const float* rstd,
                          const float* gamma, float* ds, int T, int H, int dtype,
                          cudaStream_t st, void* ds_act) {
  unsigned grid = blocks_for((int64_t)T * 32, 256);
  if (const int V = row_vec(H)) {
    if (dtype == DT_BF16) RA_VEC_SWITCH(V, ((void)launch_pdl(layernorm_bwd_vec_kernel<bf16, VV>, dim3(grid), dim3(256), (size_t)0, st, dy, dy2, xhat, rstd, gamma, ds, ds_act, T, H)))
    else RA_VEC_SWITCH(V, ((void)launch_pdl(layernorm_bwd_vec_kernel<float, VV>, dim3(grid), dim3(256), (size_t)0, st, dy, dy2, xhat, rstd, gamma, ds, ds_act, T, H)))
  } else if (dtype == DT_BF16) {
    layernorm_bwd_kernel<bf16><<<grid, 256, 0, st>>>(dy, dy2, xhat, rstd, gamma, ds, ds_act, T, H);
  } else {
    layernorm_bwd_kernel<float><<<grid, 256, 0, st>>>(dy, dy2, xhat, rstd, gamma, ds, ds_act, T, H);
  }
  note_launch(1);
  return cudaGetLastError();
}

cudaError_t add_layernorm_fwd(const void* x, const void* a, const float* gamma, const float* beta,
                              float eps, void* y, void* xhat, float* rstd, int T, int H, int dtype,
                              cudaStream_t st) {
  unsigned grid = blocks_for((int64_t)T * 32, 256);
  if (const int V = row_vec(H)) {
    if (dtype == DT_BF16) RA_VEC_SWITCH(V, ((void)launch_pdl(add_layernorm_fwd_vec_kernel<bf16, VV>, dim3(grid), dim3(256), (size_t)0, st, x, a, gamma, beta, eps, y, xhat, rstd, T, H)))
    else RA_VEC_SWITCH(V, ((void)launch_pdl(add_layernorm_fwd_vec_kernel<float, VV>, dim3(grid), dim3(256), (size_t)0, st, x, a, gamma, beta, eps, y, xhat, rstd, T, H)))
  } else if (dtype == DT_BF16) {
    add_layernorm_fwd_kernel<bf16><<<grid, 256, 0, st>>>(x, a, gamma, beta, eps, y, xhat, rstd, T, H);
  } else {
    add_layernorm_fwd_kernel<float><<<grid, 256, 0, st>>>(x, a, gamma, beta, eps, y, xhat, rstd, T, H);
  }
  note_launch(1);
  return cudaGetLastError();
}

cudaError_t rmsnorm_fwd(const void* x, int x_dtype, const float* gamma, float eps, void* n,
                        int n_dtype, float* rstd, float* x_f32_out, int T, int H,
                        cudaStream_t st) {
  unsigned grid = blocks_for((int64_t)T * 32, 256);
  if (const int V = row_vec(H)) {
    if (x_dtype == DT_BF16 && n_dtype == DT_BF16)
      RA_VEC_SWITCH(V, ((void)launch_pdl(rmsnorm_fwd_vec_kernel<bf16, bf16, VV>, dim3(grid), dim3(256), (size_t)0, st, x, gamma, eps, n, rstd, x_f32_out, T, H)))
    else if (x_dtype == DT_F32 && n_dtype == DT_BF16)
      RA_VEC_SWITCH(V, ((void)launch_pdl(rmsnorm_fwd_vec_kernel<float, bf16, VV>, dim3(grid), dim3(256), (size_t)0, st, x, gamma, eps, n, rstd, x_f32_out, T, H)))
    else if (x_dtype == DT_BF16)
      RA_VEC_SWITCH(V, ((void)launch_pdl(rmsnorm_fwd_vec_kernel<bf16, float, VV>, dim3(grid), dim3(256), (size_t)0, st, x, gamma, eps, n, rstd, x_f32_out, T, H)))
    else
      RA_VEC_SWITCH(V, ((void)launch_pdl(rmsnorm_fwd_vec_kernel<float, float, VV>, dim3(grid), dim3(256), (size_t)0, st, x, gamma, eps, n, rstd, x_f32_out, T, H)))
    note_launch(1);
    return cudaGetLastError();
  }
  if (x_dtype == DT_BF16 && n_dtype == DT_BF16)
    rmsnorm_fwd_kernel<bf16, bf16><<<grid, 256, 0, st>>>(x, gamma, eps, n, rstd, x_f32_out, T, H);
  else if (x_dtype == DT_F32 && n_dtype == DT_BF16)
    rmsnorm_fwd_kernel<float, bf16><<<grid, 256, 0, st>>>(x, gamma, eps, n, rstd, x_f32_out, T, H);
  else if (x_dtype == DT_BF16)
    rmsnorm_fwd_kernel<bf16, float><<<grid, 256, 0, st>>>(x, gamma, eps, n, rstd, x_f32_out, T, H);
  else
    rmsnorm_fwd_kernel<float, float><<<grid, 256, 0, st>>>(x, gamma, eps, n, rstd, x_f32_out, T, H);
  note_launch(1);
  return cudaGetLastError();
}

cudaError_t rmsnorm_bwd(const float* dy, const float* x, const float* rstd, const float* gamma,
                        const float* resid, float* dx, int T, int H, cudaStream_t st) {
  if (const int V = row_vec(H))
    RA_VEC_SWITCH(V, ((void)launch_pdl(rmsnorm_bwd_vec_kernel<VV>, dim3(blocks_for((int64_t)T * 32, 256)), dim3(256), (size_t)0, st, dy, x, rstd, gamma, resid, dx, T, H)))
  else
    rmsnorm_bwd_kernel<<<blocks_for((int64_t)T * 32, 256), 256, 0, st>>>(dy, x, rstd, gamma, resid, dx, T, H);
  note_launch(1);
  return cudaGetLastError();
}

cudaError_t encoder_head_fwd(const void* y, int dtype, const float* Wh, const float* bh,
                             const int32_t* labels, int B, int S, int H, int C, float* loss,
                             float* logits_out, float* dlogits, unsigned* err, cudaStream_t st) {
  if (C > MAXC || B > MAXB) return cudaErrorInvalidValue;
  auto k = dtype == DT_BF16 ? (C <= 2 ? encoder_head_fwd_kernel<bf16, 2>
                               : C <= 8 ? encoder_head_fwd_kernel<bf16, 8> : encoder_head_fwd_kernel<bf16, MAXC>)
                            : (C <= 2 ? encoder_head_fwd_kernel<float, 2>
                               : C <= 8 ? encoder_head_fwd_kernel<float, 8> : encoder_head_fwd_kernel<float, MAXC>);
  k<<<1, HEAD_FWD_THREADS, 0, st>>>(y, Wh, bh, labels, B, S, H, C, loss, logits_out, dlogits, err);
  note_launch(1);
  return cudaGetLastError();
}

cudaError_t encoder_head_bwd(const void* y, int dtype, const float* Wh, const float* dlogits,
                             int B, int S, int H, int C, float* dWh, float* dbh, float* dy,
                             cudaStream_t st) {
  if (C > MAXC || B > MAXB) return cudaErrorInvalidValue;
  unsigned grid = blocks_for(H, HEAD_BWD_THREADS);
  auto k = dtype == DT_BF16 ? (C <= 2 ? encoder_head_bwd_kernel<bf16, 2>
                               : C <= 8 ? encoder_head_bwd_kernel<bf16, 8> : encoder_head_bwd_kernel<bf16, MAXC>)
                            : (C <= 2 ? encoder_head_bwd_kernel<float, 2>
                               : C <= 8 ? encoder_head_bwd_kernel<float, 8> : encoder_head_bwd_kernel<float, MAXC>);
  k<<<grid, HEAD_BWD_THREADS, 0, st>>>(y, Wh, dlogits, B, S, H, C, dWh, dbh, dy);
  note_launch(1);
  return cudaGetLastError();
}

int span_head_chunks() { return SPAN_CHUNKS; }

cudaError_t span_head_fwd(const void* y, int dtype, const float* Wh, const float* bh,
                          const int32_t* labels, int B, int S, int H, float* row_loss, float* loss,
                          float* logits_out, float* dlogits, unsigned* err, cudaStream_t st) {
  if (S < 1 || S > SPAN_MAX_SEQ || B < 1 || H % 8) return cudaErrorInvalidValue;
  const int T = B * S;
  cudaError_t e = dtype == DT_BF16
      ? launch_pdl(span_head_logits_kernel<bf16>, dim3(blocks_for(T, 8)), dim3(256), (size_t)0, st, y, Wh, bh, T, H, dlogits)
      : launch_pdl(span_head_logits_kernel<float>, dim3(blocks_for(T, 8)), dim3(256), (size_t)0, st, y, Wh, bh, T, H, dlogits);
  if (e != cudaSuccess) return e;
  e = launch_pdl(span_head_ce_kernel, dim3(B), dim3(64), (size_t)0, st, labels, B, S, row_loss, logits_out, dlogits, err);
  if (e != cudaSuccess) return e;
  mean_kernel<<<1, 256, 0, st>>>(row_loss, B, loss);
  note_launch(3);
  return cudaGetLastError();
}

cudaError_t span_head_bwd(const void* y, int dtype, const float* Wh, const float* dlogits, int B,
                          int S, int H, float* dWh, float* dbh, float* dy, float* part,
                          cudaStream_t st) {
  if (H % 4) return cudaErrorInvalidValue;
  const int T = B * S;
  span_head_dy_kernel<<<blocks_for((int64_t)T, 8), 256, 0, st>>>(Wh, dlogits, T, H, dy);
  note_launch(1);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess || (!dWh && !dbh)) return e;
  const int chunk = (T + SPAN_CHUNKS - 1) / SPAN_CHUNKS;
  float* part_b = part + (size_t)SPAN_CHUNKS * 2 * H;
  dim3 grid(blocks_for(H, 128), SPAN_CHUNKS);
  if (dtype == DT_BF16)
    span_head_dw_kernel<bf16><<<grid, 128, 0, st>>>(y, dlogits, T, H, chunk, part, part_b);
  else
    span_head_dw_kernel<float><<<grid, 128, 0, st>>>(y, dlogits, T, H, chunk, part, part_b);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  span_head_dw_reduce_kernel<<<blocks_for((int64_t)2 * H, 256), 256, 0, st>>>(part, part_b, SPAN_CHUNKS, H, dWh, dbh);
  note_launch(2);
  return cudaGetLastError();
}

cudaError_t vocab_ce(void* logits, int dtype, int ld, const int32_t* labels, int T, int V,
                     float* row_loss, float* loss, float* logits_out, unsigned* err,
                     cudaStream_t st) {
  if (dtype == DT_BF16)
    vocab_ce_kernel<bf16><<<T, 256, 0, st>>>(logits, ld, labels, T, V, row_loss, logits_out, err);
  else
    vocab_ce_kernel<float><<<T, 256, 0, st>>>(logits, ld, labels, T, V, row_loss, logits_out, err);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  mean_kernel<<<1, 256, 0, st>>>(row_loss, T, loss);
  note_launch(2);
  return cudaGetLastError();
}

cudaError_t adam_update(const AdamArgs& a, cudaStream_t st) {
  if (a.n <= 0) return cudaSuccess;
  adam_kernel<<<blocks_for(a.n, 256), 256, 0, st>>>(a);
  note_launch(1);
  return cudaGetLastError();
}

cudaError_t adam_bump(int32_t* steps, int n, cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  bump_kernel<<<blocks_for(n, 128), 128, 0, st>>>(steps, n);
  note_launch(1);
  return cudaGetLastError();
}

cudaError_t convert_f32(const float* src, void* dst, int dst_dtype, int64_t n, cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  if (dst_dtype == DT_BF16) convert_kernel<bf16><<<blocks_for(n, 256), 256, 0, st>>>(src, dst, n);
  else convert_kernel<float><<<blocks_for(n, 256), 256, 0, st>>>(src, dst, n);
  note_launch(1);
  return cudaGetLastError();
}

cudaError_t transpose_f32(const float* src, void* dst, int dst_dtype, int rows, int cols,
                          int ld_dst, cudaStream_t st) {
  dim3 grid((cols + 31) / 32, (rows + 31) / 32), blk(32, 8);
  if (dst_dtype == DT_BF16) transpose_kernel<bf16><<<grid, blk, 0, st>>>(src, dst, rows, cols, ld_dst);
  else transpose_kernel<float><<<grid, blk, 0, st>>>(src, dst, rows, cols, ld_dst);
  note_launch(1);
  return cudaGetLastError();
}

cudaError_t pack_rows(const float* src, void* dst, int dst_dtype, int R, int C, int part,
                      bool transposed, cudaStream_t st) {
  int64_t n = (int64_t)R * C;
  if (dst_dtype == DT_BF16) pack_rows_kernel<bf16><<<blocks_for(n, 256), 256, 0, st>>>(src, dst, R, C, part, transposed);
  else pack_rows_kernel<float><<<blocks_for(n, 256), 256, 0, st>>>(src, dst, R, C, part, transposed);
  note_launch(1);
  return cudaGetLastError();
}

cudaError_t adapter_transpose(const float* P, float* PT, void* PB, void* PTB, int n_layers,
                              int H, int m, cudaStream_t st) {
  if (n_layers <= 0) return cudaSuccess;
  // both orientations of a matrix hold the same number of 32 x 32 tiles
  dim3 grid((unsigned)(((H + 31) / 32) * ((m + 31) / 32)), 1, 4 * n_layers);
  adapter_transpose_kernel<<<grid, 256, 0, st>>>(P, PT, reinterpret_cast<bf16*>(PB),
                                                 reinterpret_cast<bf16*>(PTB), H, m);
  note_launch(1);
  return cudaGetLastError();
}

cudaError_t adam_adapter_update(const AdamArgs& a, float* PT, void* PB, void* PTB, int n_layers,
                                int H, int m, cudaStream_t st) {
  if (n_layers <= 0) return cudaSuccess;
  dim3 grid((unsigned)(((H + 31) / 32) * ((m + 31) / 32)), 1, 4 * n_layers);
  adam_adapter_kernel<<<grid, 256, 0, st>>>(a, PT, reinterpret_cast<bf16*>(PB), reinterpret_cast<bf16*>(PTB),
                                            H, m);
  note_launch(1);
  return cudaGetLastError();
}

cudaError_t eval_activation(int which, const float* x, float* y, int64_t n, cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  activation_kernel<<<blocks_for(n, 256), 256, 0, st>>>(which, x, y, n);
  note_launch(1);
  return cudaGetLastError();
}

cudaError_t fill_f32(float* dst, float v, int64_t n, cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  fill_kernel<<<blocks_for(n, 256), 256, 0, st>>>(dst, v, n);
  note_launch(1);
  return cudaGetLastError();
}

}  // namespace ra
