// k_attention.cu -- fused attention forward and backward (CUDA-core version).
//
// softmax(q k^T * scale [+ causal mask]) v per (batch, head), with the online softmax so
// the S x S score matrix never reaches memory.  The forward saves the row log-sum-exp;
// the backward recomputes P from q, k and that statistic (no P is stored).  RoPE
// (rotate-half, pairs (i, i + dh/2)) is applied to q and k as they are loaded, and its
// transpose to dq and dk as they are stored, so the saved q|k|v are the raw projections.
// The backward is two deterministic kernels: dK/dV with the keys held and the queries
// streamed, and dQ with the queries held and the keys streamed.
#include "common.cuh"
#include "kernels.h"

namespace ra {
namespace {

constexpr int QB = 64;   // queries per CTA (forward)
constexpr int KB = 64;   // keys per smem block
constexpr int MAXD = 128;

template <typename T>
__device__ __forceinline__ float ldv(const T* p, int64_t i) { return to_f(p[i]); }

__device__ __forceinline__ float rope_inv_freq(int i, int dh, float theta) {
  // theta^(-2i/dh)
  return expf(-logf(theta) * (2.0f * (float)i / (float)dh));
}

// Loads rows [r0, r0+n) of one head's q, k or v (column offset col0 in the [T, 3H] qkv)
// into smem as float [n][ld], applying RoPE if asked.  Rows beyond S are zero.
template <typename T>
__device__ void load_rows(float* dst, int ld, const T* qkv, int ld_qkv, int b, int S, int r0,
                          int n, int col0, int dh, bool rope, float theta) {
  for (int e = threadIdx.x; e < n * dh; e += blockDim.x) {
    int r = e / dh, d = e % dh;
    int s = r0 + r;
    dst[r * ld + d] = (s < S) ? ldv(qkv, (int64_t)(b * S + s) * ld_qkv + col0 + d) : 0.f;
  }
  if (!rope) return;
  __syncthreads();
  int half = dh / 2;
  for (int e = threadIdx.x; e < n * half; e += blockDim.x) {
    int r = e / half, i = e % half;
    int s = r0 + r;
    float sn, cs;
    sincosf((float)s * rope_inv_freq(i, dh, theta), &sn, &cs);
    float x1 = dst[r * ld + i], x2 = dst[r * ld + i + half];
    dst[r * ld + i] = x1 * cs - x2 * sn;
    dst[r * ld + i + half] = x2 * cs + x1 * sn;
  }
}

// ---------------------------------------------------------------------------------------
// forward: CTA = (64 queries, one (b, head)); warp w owns queries w*8 .. w*8+7
// ---------------------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(256) attn_fwd_kernel(AttnArgs a) {
  extern __shared__ float sm[];
  const int dh = a.head_dim, ld = dh + 1;
  float* Qs = sm;               // [QB][ld]
  float* Ks = Qs + QB * ld;     // [KB][ld]
  float* Vs = Ks + KB * ld;     // [KB][ld]
  const int bh = blockIdx.y, b = bh / a.n_heads, hh = bh % a.n_heads;
  const int H = a.n_heads * dh, ld_qkv = 3 * H;
  const int q0 = blockIdx.x * QB;
  const T* qkv = reinterpret_cast<const T*>(a.qkv);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nd = dh / 32;  // dims per lane (dh in {32, 64, 96, 128})

  load_rows<T>(Qs, ld, qkv, ld_qkv, b, a.S, q0, QB, hh * dh, dh, a.rope, a.rope_theta);

  float o[8][4], mrow[8], lrow[8];
#pragma unroll
  for (int qi = 0; qi < 8; ++qi) {
    mrow[qi] = -INFINITY; lrow[qi] = 0.f;
#pragma unroll
    for (int c = 0; c < 4; ++c) o[qi][c] = 0.f;
  }
  int kend = a.causal ? min(a.S, q0 + QB) : a.S;
  for (int k0 = 0; k0 < kend; k0 += KB) {
    __syncthreads();
    load_rows<T>(Ks, ld, qkv, ld_qkv, b, a.S, k0, KB, H + hh * dh, dh, a.rope, a.rope_theta);
    load_rows<T>(Vs, ld, qkv, ld_qkv, b, a.S, k0, KB, 2 * H + hh * dh, dh, false, 0.f);
    __syncthreads();
#pragma unroll 1
    for (int qi = 0; qi < 8; ++qi) {
      int ql = warp * 8 + qi, q = q0 + ql;
      if (q >= a.S) break;
      float s[2];
#pragma unroll
      for (int jj = 0; jj < 2; ++jj) {
        int kl = lane + 32 * jj, key = k0 + kl;
        float acc = 0.f;
        for (int d = 0; d < dh; ++d) acc = fmaf(Qs[ql * ld + d], Ks[kl * ld + d], acc);
        bool valid = key < a.S && (!a.causal || key <= q);
        s[jj] = valid ? acc * a.scale : -INFINITY;
      }
      float mb = warp_max(fmaxf(s[0], s[1]));
      float mnew = fmaxf(mrow[qi], mb);
      if (mnew == -INFINITY) continue;  // no valid key yet
      float alpha = expf(mrow[qi] - mnew);
      float p0 = expf(s[0] - mnew), p1 = expf(s[1] - mnew);
      lrow[qi] = lrow[qi] * alpha + warp_sum(p0 + p1);
      mrow[qi] = mnew;
#pragma unroll
      for (int c = 0; c < 4; ++c) o[qi][c] *= alpha;
      for (int j = 0; j < KB; ++j) {
        float pj = __shfl_sync(0xffffffffu, j < 32 ? p0 : p1, j & 31);
#pragma unroll
        for (int c = 0; c < 4; ++c)
          if (c < nd) o[qi][c] = fmaf(pj, Vs[j * ld + lane + 32 * c], o[qi][c]);
      }
    }
  }
  T* O = reinterpret_cast<T*>(a.O);
#pragma unroll
  for (int qi = 0; qi < 8; ++qi) {
    int q = q0 + warp * 8 + qi;
    if (q >= a.S) break;
    float inv = 1.f / lrow[qi];
    int64_t row = (int64_t)(b * a.S + q) * H + hh * dh;
#pragma unroll
    for (int c = 0; c < 4; ++c)
      if (c < nd) O[row + lane + 32 * c] = from_f<T>(o[qi][c] * inv);
    if (a.lse && lane == 0) a.lse[(int64_t)bh * a.S + q] = mrow[qi] + logf(lrow[qi]);
  }
}

// D[b, h, s] = sum_d dO * O  (one warp per (token, head))
template <typename T>
__global__ void attn_bwd_pre_kernel(AttnArgs a) {
  pdl_wait();
  pdl_trigger();
  int gw = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  int T_ = a.B * a.S;
  if (gw >= T_ * a.n_heads) return;
  int t = gw / a.n_heads, hh = gw % a.n_heads;
  int b = t / a.S, s = t % a.S;
  int dh = a.head_dim, H = a.n_heads * dh;
  const T* O = reinterpret_cast<const T*>(a.O);
  const T* dO = reinterpret_cast<const T*>(a.dO);
  float acc = 0.f;
  for (int d = lane; d < dh; d += 32) {
    int64_t i = (int64_t)t * H + hh * dh + d;
    acc += to_f(O[i]) * to_f(dO[i]);
  }
  acc = warp_sum(acc);
  if (lane == 0) a.Dscratch[((int64_t)b * a.n_heads + hh) * a.S + s] = acc;
}

// bf16, head_dim 64 or 128: G = head_dim / 8 threads per (token, head), 16-byte loads
template <int G>
__global__ void __launch_bounds__(256) attn_bwd_pre_vec_kernel(AttnArgs a) {
  pdl_wait();
  pdl_trigger();
  const int64_t gi = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) / G;
  const int r = threadIdx.x % G;
  const int T_ = a.B * a.S;
  // groups past the end stay for the shuffles below (full warps) but touch no memory
  const bool live = gi < (int64_t)T_ * a.n_heads;
  const int t = live ? (int)(gi / a.n_heads) : 0, hh = live ? (int)(gi % a.n_heads) : 0;
  const int b = t / a.S, s = t % a.S;
  const int dh = 8 * G, H = a.n_heads * dh;
  const int64_t i = (int64_t)t * H + hh * dh + 8 * r;
  uint4 o = make_uint4(0, 0, 0, 0), g = o;
  if (live) {
    o = __ldg(reinterpret_cast<const uint4*>(reinterpret_cast<const bf16*>(a.O) + i));
    g = __ldg(reinterpret_cast<const uint4*>(reinterpret_cast<const bf16*>(a.dO) + i));
  }
  const __nv_bfloat162* o2 = reinterpret_cast<const __nv_bfloat162*>(&o);
  const __nv_bfloat162* g2 = reinterpret_cast<const __nv_bfloat162*>(&g);
  float acc = 0.f;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const float2 x = __bfloat1622float2(o2[k]), y = __bfloat1622float2(g2[k]);
    acc += x.x * y.x + x.y * y.y;
  }
#pragma unroll
  for (int off = G / 2; off > 0; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
  if (live && r == 0) a.Dscratch[((int64_t)b * a.n_heads + hh) * a.S + s] = acc;
}

// thread-group layout of the backward: 8 threads per key (or query); thread r of a group
// owns dims r, r+8, r+16, ... so both members of every RoPE pair (d, d + dh/2) stay in it.
constexpr int GRP = 8;
constexpr int DPT = MAXD / GRP;  // 16 dims per thread max

__device__ __forceinline__ float grp_sum(float v) {
  v += __shfl_xor_sync(0xffffffffu, v, 1);
  v += __shfl_xor_sync(0xffffffffu, v, 2);
  v += __shfl_xor_sync(0xffffffffu, v, 4);
  return v;
}

// un-rotate a gradient held by one thread group member (dims r + 8c) for position s
__device__ __forceinline__ void rope_bwd_regs(float* g, int r, int dh, int s, float theta) {
  int half = dh / 2, npt = dh / GRP;
  for (int c = 0; c < npt / 2; ++c) {
    int i = r + GRP * c;  // < half
    float sn, cs;
    sincosf((float)s * rope_inv_freq(i, dh, theta), &sn, &cs);
    int c2 = c + half / GRP;
    float d1 = g[c], d2 = g[c2];
    g[c] = d1 * cs + d2 * sn;
    g[c2] = d2 * cs - d1 * sn;
  }
}

// dK, dV: CTA = (32 keys, one (b, head)); 8 threads per key; queries streamed in blocks
template <typename T>
__global__ void __launch_bounds__(256) attn_bwd_dkdv_kernel(AttnArgs a) {
  extern __shared__ float sm[];
  const int dh = a.head_dim, ld = dh + 1;
  constexpr int NK = 32, NQ = 64;
  float* Qs = sm;             // [NQ][ld]
  float* dOs = Qs + NQ * ld;  // [NQ][ld]
  float* Ls = dOs + NQ * ld;  // [NQ] lse
  float* Ds = Ls + NQ;        // [NQ]
  float* Kst = Ds + NQ;       // [NK][ld] staging of this CTA's keys/values
  float* Vst = Kst + NK * ld;
  const int bh = blockIdx.y, b = bh / a.n_heads, hh = bh % a.n_heads;
  const int H = a.n_heads * dh, ld_qkv = 3 * H;
  const int k0 = blockIdx.x * NK;
  const T* qkv = reinterpret_cast<const T*>(a.qkv);
  const T* dO = reinterpret_cast<const T*>(a.dO);
  const int kl = threadIdx.x / GRP, r = threadIdx.x % GRP, key = k0 + kl;
  const int npt = dh / GRP;

  load_rows<T>(Kst, ld, qkv, ld_qkv, b, a.S, k0, NK, H + hh * dh, dh, a.rope, a.rope_theta);
  load_rows<T>(Vst, ld, qkv, ld_qkv, b, a.S, k0, NK, 2 * H + hh * dh, dh, false, 0.f);
  __syncthreads();
  float kr[DPT], vr[DPT], dk[DPT], dv[DPT];
#pragma unroll
  for (int c = 0; c < DPT; ++c) {
    bool in = c < npt;
    kr[c] = in ? Kst[kl * ld + r + GRP * c] : 0.f;
    vr[c] = in ? Vst[kl * ld + r + GRP * c] : 0.f;
    dk[c] = 0.f; dv[c] = 0.f;
  }
  int qstart = a.causal ? k0 : 0;
  for (int q0 = (qstart / NQ) * NQ; q0 < a.S; q0 += NQ) {
    __syncthreads();
    load_rows<T>(Qs, ld, qkv, ld_qkv, b, a.S, q0, NQ, hh * dh, dh, a.rope, a.rope_theta);
    for (int e = threadIdx.x; e < NQ * dh; e += blockDim.x) {
      int rr = e / dh, d = e % dh, s = q0 + rr;
      dOs[rr * ld + d] = s < a.S ? to_f(dO[(int64_t)(b * a.S + s) * H + hh * dh + d]) : 0.f;
    }
    for (int e = threadIdx.x; e < NQ; e += blockDim.x) {
      int s = q0 + e;
      Ls[e] = s < a.S ? a.lse[(int64_t)bh * a.S + s] : 0.f;
      Ds[e] = s < a.S ? a.Dscratch[(int64_t)bh * a.S + s] : 0.f;
    }
    __syncthreads();
    for (int qi = 0; qi < NQ; ++qi) {
      int q = q0 + qi;
      if (q >= a.S) break;
      float sp = 0.f, dpp = 0.f;
#pragma unroll
      for (int c = 0; c < DPT; ++c) {
        if (c < npt) {
          sp = fmaf(Qs[qi * ld + r + GRP * c], kr[c], sp);
          dpp = fmaf(dOs[qi * ld + r + GRP * c], vr[c], dpp);
        }
      }
      sp = grp_sum(sp);
      dpp = grp_sum(dpp);
      bool valid = key < a.S && (!a.causal || key <= q);
      float p = valid ? expf(sp * a.scale - Ls[qi]) : 0.f;
      float ds = p * (dpp - Ds[qi]) * a.scale;
#pragma unroll
      for (int c = 0; c < DPT; ++c) {
        if (c < npt) {
          dv[c] = fmaf(p, dOs[qi * ld + r + GRP * c], dv[c]);
          dk[c] = fmaf(ds, Qs[qi * ld + r + GRP * c], dk[c]);
        }
      }
    }
  }
  if (key >= a.S) return;
  if (a.rope) rope_bwd_regs(dk, r, dh, key, a.rope_theta);
  T* dqkv = reinterpret_cast<T*>(a.dqkv);
  int64_t row = (int64_t)(b * a.S + key) * ld_qkv;
  for (int c = 0; c < npt; ++c) {
    dqkv[row + H + hh * dh + r + GRP * c] = from_f<T>(dk[c]);
    dqkv[row + 2 * H + hh * dh + r + GRP * c] = from_f<T>(dv[c]);
  }
}

// dQ: CTA = (32 queries, one (b, head)); 8 threads per query; keys streamed in blocks
template <typename T>
__global__ void __launch_bounds__(256) attn_bwd_dq_kernel(AttnArgs a) {
  extern __shared__ float sm[];
  const int dh = a.head_dim, ld = dh + 1;
  constexpr int NQ = 32;
  float* Ks = sm;            // [KB][ld]
  float* Vs = Ks + KB * ld;  // [KB][ld]
  float* Qst = Vs + KB * ld; // [NQ][ld]
  float* dOst = Qst + NQ * ld;
  const int bh = blockIdx.y, b = bh / a.n_heads, hh = bh % a.n_heads;
  const int H = a.n_heads * dh, ld_qkv = 3 * H;
  const int q0 = blockIdx.x * NQ;
  const T* qkv = reinterpret_cast<const T*>(a.qkv);
  const T* dO = reinterpret_cast<const T*>(a.dO);
  const int ql = threadIdx.x / GRP, r = threadIdx.x % GRP, q = q0 + ql;
  const int npt = dh / GRP;

  load_rows<T>(Qst, ld, qkv, ld_qkv, b, a.S, q0, NQ, hh * dh, dh, a.rope, a.rope_theta);
  for (int e = threadIdx.x; e < NQ * dh; e += blockDim.x) {
    int rr = e / dh, d = e % dh, s = q0 + rr;
    dOst[rr * ld + d] = s < a.S ? to_f(dO[(int64_t)(b * a.S + s) * H + hh * dh + d]) : 0.f;
  }
  __syncthreads();
  float qr[DPT], dor[DPT], dq[DPT];
#pragma unroll
  for (int c = 0; c < DPT; ++c) {
    bool in = c < npt;
    qr[c] = in ? Qst[ql * ld + r + GRP * c] : 0.f;
    dor[c] = in ? dOst[ql * ld + r + GRP * c] : 0.f;
    dq[c] = 0.f;
  }
  float lse = q < a.S ? a.lse[(int64_t)bh * a.S + q] : 0.f;
  float Dq = q < a.S ? a.Dscratch[(int64_t)bh * a.S + q] : 0.f;
  int kend = a.causal ? min(a.S, q0 + NQ) : a.S;
  for (int k0 = 0; k0 < kend; k0 += KB) {
    __syncthreads();
    load_rows<T>(Ks, ld, qkv, ld_qkv, b, a.S, k0, KB, H + hh * dh, dh, a.rope, a.rope_theta);
    load_rows<T>(Vs, ld, qkv, ld_qkv, b, a.S, k0, KB, 2 * H + hh * dh, dh, false, 0.f);
    __syncthreads();
    for (int j = 0; j < KB; ++j) {
      int key = k0 + j;
      if (key >= a.S) break;
      float sp = 0.f, dpp = 0.f;
#pragma unroll
      for (int c = 0; c < DPT; ++c) {
        if (c < npt) {
          sp = fmaf(qr[c], Ks[j * ld + r + GRP * c], sp);
          dpp = fmaf(dor[c], Vs[j * ld + r + GRP * c], dpp);
        }
      }
      sp = grp_sum(sp);
      dpp = grp_sum(dpp);
      bool valid = q < a.S && (!a.causal || key <= q);
      float p = valid ? expf(sp * a.scale - lse) : 0.f;
      float ds = p * (dpp - Dq) * a.scale;
#pragma unroll
      for (int c = 0; c < DPT; ++c)
        if (c < npt) dq[c] = fmaf(ds, Ks[j * ld + r + GRP * c], dq[c]);
    }
  }
  if (q >= a.S) return;
  if (a.rope) rope_bwd_regs(dq, r, dh, q, a.rope_theta);
  T* dqkv = reinterpret_cast<T*>(a.dqkv);
  int64_t row = (int64_t)(b * a.S + q) * ld_qkv;
  for (int c = 0; c < npt; ++c) dqkv[row + hh * dh + r + GRP * c] = from_f<T>(dq[c]);
}

template <typename T>
cudaError_t fwd_impl(const AttnArgs& a, cudaStream_t st) {
  int ld = a.head_dim + 1;
  size_t smem = (size_t)(QB + 2 * KB) * ld * sizeof(float);
  cudaFuncSetAttribute(attn_fwd_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  dim3 grid((a.S + QB - 1) / QB, a.B * a.n_heads);
  attn_fwd_kernel<T><<<grid, 256, smem, st>>>(a);
  note_launch(1);
  return cudaGetLastError();
}

template <typename T>
cudaError_t bwd_impl(const AttnArgs& a, cudaStream_t st) {
  int T_ = a.B * a.S;
  int64_t warps = (int64_t)T_ * a.n_heads;
  cudaError_t le;
  if (a.dtype == DT_BF16 && (a.head_dim == 64 || a.head_dim == 128)) {
    const int G = a.head_dim / 8;
    const unsigned blocks = (unsigned)((warps * G + 255) / 256);
    le = G == 8 ? launch_pdl(attn_bwd_pre_vec_kernel<8>, dim3(blocks), dim3(256), (size_t)0, st, a)
                : launch_pdl(attn_bwd_pre_vec_kernel<16>, dim3(blocks), dim3(256), (size_t)0, st, a);
  } else {
    le = launch_pdl(attn_bwd_pre_kernel<T>, dim3((unsigned)((warps * 32 + 255) / 256)), dim3(256),
                    (size_t)0, st, a);
  }
  note_launch(1);
  if (le != cudaSuccess) return le;
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  if (attention_mma_ok(a)) return attention_bwd_mma(a, st);
  int ld = a.head_dim + 1;
  size_t smem1 = (size_t)(2 * 64 * ld + 2 * 64 + 2 * 32 * ld) * sizeof(float);
  cudaFuncSetAttribute(attn_bwd_dkdv_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem1);
  attn_bwd_dkdv_kernel<T><<<dim3((a.S + 31) / 32, a.B * a.n_heads), 256, smem1, st>>>(a);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  size_t smem2 = (size_t)(2 * KB * ld + 2 * 32 * ld) * sizeof(float);
  cudaFuncSetAttribute(attn_bwd_dq_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem2);
  attn_bwd_dq_kernel<T><<<dim3((a.S + 31) / 32, a.B * a.n_heads), 256, smem2, st>>>(a);
  note_launch(2);
  return cudaGetLastError();
}

}  // namespace

cudaError_t attention_fwd(const AttnArgs& a, cudaStream_t st) {
  if (a.head_dim > MAXD || a.head_dim % 32 != 0) return cudaErrorInvalidValue;
  if (attention_mma_ok(a)) return attention_fwd_mma(a, st);
  return a.dtype == DT_BF16 ? fwd_impl<bf16>(a, st) : fwd_impl<float>(a, st);
}

cudaError_t attention_bwd(const AttnArgs& a, cudaStream_t st) {
  if (a.head_dim > MAXD || a.head_dim % 32 != 0) return cudaErrorInvalidValue;
  return a.dtype == DT_BF16 ? bwd_impl<bf16>(a, st) : bwd_impl<float>(a, st);
}

}  // namespace ra
