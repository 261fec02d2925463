// kernels.h -- host-side launchers of the libringada kernels (internal, not ABI).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace ra {

enum DType : int { DT_F32 = 0, DT_BF16 = 1 };

inline size_t dtype_size(int dt) { return dt == DT_BF16 ? 2 : 4; }

// Launches kernel k with programmatic stream serialisation: it may start while the previous
// kernel of the stream finishes, and must call pdl_wait() before touching memory that earlier
// kernels use.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*k)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t st, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, k, args...);
}

// Counts kernels launched by this library (process-wide), for launch accounting.
void note_launch(int n);
long long launches_so_far();

// ---------------------------------------------------------------------------------------
// GEMM  C[M, N] = A[M, K] * B[N, K]^T with a fused epilogue.  A and B share a dtype and are
// K-major (row-major, K contiguous).  The accumulator is fp32.
// ---------------------------------------------------------------------------------------
enum EpiKind : int {
  EPI_STORE = 0,     // C = acc (+ bias)
  EPI_BIAS_GELU,     // C = acc + bias (pre-activation u, optional), C2 = GELU(u)
  EPI_MUL,           // C = acc * aux                  (aux = GELU'(u) saved by BIAS_GELU_G)
  EPI_RESID,         // C = acc + aux                  (aux = fp32 residual)
  EPI_DSWIGLU,       // N = F: acc is d(h) at col j; aux = packed [gate|up] [M, 2F];
                     // C (width 2F, packed like aux) gets d(gate), d(up)
  EPI_SWIGLU,        // N = 2F packed [gate|up]: C = packed pre-activations (optional),
                     // C2 [M, F] = silu(gate) * up
  EPI_BIAS_GELU_G,   // u = acc + bias: C = GELU'(u) (optional), C2 = GELU(u) -- the factor the
                     // backward multiplies by (EPI_MUL), evaluated once in the forward
};

struct GemmArgs {
  const void* A = nullptr; int lda = 0;
  // B is [N, K] (K contiguous) by default; with b_kn it is read as stored [K, N] (N
  // contiguous, ldb = its row stride): the dX GEMMs multiply by a forward weight [out, in]
  // without a transposed copy
  const void* B = nullptr; int ldb = 0;
  bool b_kn = false;
  int M = 0, N = 0, K = 0;
  int in_dtype = DT_F32;
  int epi = EPI_STORE;
  void* C = nullptr; int ldc = 0; int c_dtype = DT_F32;
  const float* bias = nullptr;
  void* C2 = nullptr; int ldc2 = 0; int c2_dtype = DT_F32;
  const void* aux = nullptr; int ldaux = 0; int aux_dtype = DT_F32;
  unsigned* err = nullptr;
  // stream-K scratch of the tcgen05 path (nullable: then every tile is done by one CTA):
  // sk_slots partial-accumulator slots of gemm_sk_slot_bytes() and sk_slots * 12 flags,
  // zero before the first launch (every launch leaves them zero).  GEMMs that may run at the
  // same time (different streams) need different scratch.
  float* sk_ws = nullptr;
  unsigned* sk_flags = nullptr;
  int sk_slots = 0;
};
// bytes of one stream-K slot, flags per slot
size_t gemm_sk_slot_bytes();
int gemm_sk_flags_per_slot();

// Returns a cudaError_t from the launch (cudaSuccess if enqueued).
cudaError_t gemm(const GemmArgs& a, cudaStream_t st);
// tcgen05 path; returns cudaErrorNotSupported if the shape/dtype is not handled.
cudaError_t gemm_tc(const GemmArgs& a, cudaStream_t st);
cudaError_t gemm_simt(const GemmArgs& a, cudaStream_t st);
// Bounded-wait self-test (failure detection): a wait that nothing satisfies runs out after
// limit_ns and sets RA_DEVERR_TIMEOUT in *err.
cudaError_t selftest_wait(unsigned* err, uint64_t limit_ns, cudaStream_t st);
// Whether the tcgen05 path is usable on the current device (sm_103).
bool tc_available();
int device_sm_count();
// TMA map of a row-major bf16 [rows, cols] matrix (row stride ld elements), boxes of
// box_cols x box_rows with the swizzle whose span is one box row (128-byte rows: the
// 128-byte swizzle the tcgen05 operand descriptors read); false if the driver refuses it.
bool tma_map_bf16(CUtensorMap* out, const void* ptr, int64_t rows, int64_t cols, int64_t ld, int box_cols,
                  int box_rows);

// ---------------------------------------------------------------------------------------
// Attention (per (batch, head); token t = b*S + s; head hh at columns hh*dh of q/k/v).
// ---------------------------------------------------------------------------------------
struct AttnArgs {
  const void* qkv = nullptr;  // [T, 3H]: q | k | v
  int B = 0, S = 0, n_heads = 0, head_dim = 0;
  int dtype = DT_F32;
  bool causal = false;
  bool rope = false;          // rotate-half RoPE on q and k inside the kernel
  bool qk_rotated = false;    // q and k in qkv already carry the rotation (rope_qk_inplace):
                              // the kernels stage them as they are, and the backward only
                              // applies the rotation's transpose to dq and dk
  float rope_theta = 10000.f;
  float scale = 1.f;
  void* O = nullptr;          // [T, H]
  float* lse = nullptr;       // [B, heads, S] (natural log, scaled scores) or null
  // backward
  const void* dO = nullptr;   // [T, H]
  float* Dscratch = nullptr;  // [B, heads, S]
  void* dqkv = nullptr;       // [T, 3H]
  unsigned* err = nullptr;
};
cudaError_t attention_fwd(const AttnArgs& a, cudaStream_t st);
cudaError_t attention_bwd(const AttnArgs& a, cudaStream_t st);
// tensor-core versions (bf16, head_dim 64 or 128); the backward expects D in a.Dscratch
bool attention_mma_ok(const AttnArgs& a);
// Rotates the q and k columns of a.qkv (bf16, head_dim 64 or 128) in place with RoPE
// (rotate-half pairs (i, i + dh/2), angle s * theta^(-2i/dh)), once per forward, so that
// every query block of the attention kernels can stage them with plain copies.
cudaError_t rope_qk_inplace(const AttnArgs& a, cudaStream_t st);
cudaError_t attention_fwd_mma(const AttnArgs& a, cudaStream_t st);
cudaError_t attention_bwd_mma(const AttnArgs& a, cudaStream_t st);
// tcgen05 forward (bf16, head_dim 64, no mask or RoPE, S <= 256)
bool attention_tc_ok(const AttnArgs& a);
cudaError_t attention_fwd_tc(const AttnArgs& a, cudaStream_t st);
// tcgen05 kernels over 128-row blocks (bf16, head_dim 64 or 128, causal or not, q and k
// plain or rotated in place): the backward (expects D = rowsum(dO * O) in a.Dscratch and the
// forward's lse) and the forward of sequences longer than one block
bool attention_bwd_tc_ok(const AttnArgs& a);
cudaError_t attention_bwd_tc(const AttnArgs& a, cudaStream_t st);
bool attention_fwd_blocks_tc_ok(const AttnArgs& a);
cudaError_t attention_fwd_blocks_tc(const AttnArgs& a, cudaStream_t st);

// ---------------------------------------------------------------------------------------
// Row-wise fused kernels
// ---------------------------------------------------------------------------------------
// Adapter forward (Eq. 1) fused with the residual add and the block's normalisation.
//   out_pre = a + GELU(a Wd) Wu, z = a Wd (saved if z != null)
//   encoder: y = LN(resid + out_pre) * g + b ; xhat, rstd saved (if non-null)
//   decoder: x_out(f32) = resid(f32) + out_pre ; n = RMSNorm(x_out) * g (act), rstd
//   no_norm (the paper's post-FFN placement): y = out_pre (act), no residual operand (the
//            residual of Eq. 1 is the adapter input a itself), no norm
struct AdapterFwdArgs {
  int T = 0, H = 0, m = 0, dtype = DT_F32;
  bool decoder = false;
  bool no_norm = false;
  const void* a = nullptr;      // [T, H] act
  const float* Wd = nullptr;    // [H, m]
  const float* Wu = nullptr;    // [m, H]
  float* z = nullptr;           // [T, m] or null
  const void* resid = nullptr;  // encoder: act [T, H]; decoder: f32 [T, H]
  const float* gamma = nullptr;
  const float* beta = nullptr;  // encoder only
  float eps = 1e-12f;
  void* y = nullptr;            // encoder: act [T, H] (LN output); decoder: act n
  float* x_out = nullptr;       // decoder: f32 residual stream out
  void* xhat = nullptr;         // encoder: act [T, H] or null
  float* rstd = nullptr;        // [T] or null
  // bf16 shadows of the adapter weights (bf16 models): W_down^T [m, H], W_up^T [H, m];
  // when given (and the shape suits), the tensor-core kernel runs
  const void* WdT_b = nullptr;
  const void* WuT_b = nullptr;
};
cudaError_t adapter_fwd(const AdapterFwdArgs& a, cudaStream_t st);
cudaError_t adapter_fwd_mma(const AdapterFwdArgs& a, const void* WdT_b, const void* WuT_b,
                            cudaStream_t st);
bool adapter_mma_ok(int H, int m);

// Adapter backward, row part: dz = (g Wu^T) * GELU'(z) -> dz (f32 [T, m]);
// dh = g + dz Wd^T -> dh (act) if non-null.  WuT [H, m] and WdT [m, H] are transposed copies.
struct AdapterBwdArgs {
  int T = 0, H = 0, m = 0, dtype = DT_F32;
  const float* g = nullptr;     // [T, H] f32
  const void* h = nullptr;      // [T, H] act (adapter input)
  const float* z = nullptr;     // [T, m]
  const float* WuT = nullptr;   // [H, m]
  const float* WdT = nullptr;   // [m, H]
  float* dz = nullptr;          // [T, m] scratch
  void* dh = nullptr;           // [T, H] act or null
  int dh_dtype = DT_F32;
  float* dWd = nullptr;         // [H, m]
  float* dWu = nullptr;         // [m, H]
  float* partials = nullptr;    // scratch, adapter_bwd_partials_floats(T, H, m)
  // bf16 shadows (bf16 models): W_up [m, H], W_down [H, m]
  const void* Wu_b = nullptr;
  const void* Wd_b = nullptr;
};
size_t adapter_bwd_partials_floats(int T, int H, int m);
cudaError_t adapter_bwd(const AdapterBwdArgs& a, cudaStream_t st);
cudaError_t adapter_bwd_mma(const AdapterBwdArgs& a, const void* Wu_b, const void* Wd_b,
                            cudaStream_t st);
// chunk count of the dW reduction (a pure function of T and H) and its fixed-order sum
int adapter_dw_chunks(int T, int H);
cudaError_t adapter_dw_reduce(const float* partials, int nchunk, int H, int m, float* dWd,
                              float* dWu, cudaStream_t st);

// LayerNorm backward with frozen gamma: ds = rstd * (gy - mean(gy) - xhat mean(gy xhat)),
// gy = (dy + dy2) * gamma.  dy, dy2 (nullable: 0) f32, xhat act, ds f32.  The second input
// lets a residual-stream gradient join here instead of in the producing GEMM's epilogue.
// ds_act (nullable): a copy of ds in the activation type, for a GEMM that reads it.
cudaError_t layernorm_bwd(const float* dy, const float* dy2, const void* xhat, const float* rstd,
                          const float* gamma, float* ds, int T, int H, int dtype,
                          cudaStream_t st, void* ds_act = nullptr);
// LayerNorm of a residual sum (the add & norm sublayer): y = LN(x + a) * gamma + beta with
// biased variance; xhat = the normalised sum and rstd = 1 / sqrt(var + eps) saved when
// non-null.  x, a, y, xhat in dtype; statistics in fp32.
cudaError_t add_layernorm_fwd(const void* x, const void* a, const float* gamma, const float* beta,
                              float eps, void* y, void* xhat, float* rstd, int T, int H, int dtype,
                              cudaStream_t st);
// RMSNorm forward: n = x * rstd * gamma; x given as act (x_act) or f32 (x_f32);
// optionally copies x into x_f32_out (f32 residual stream).
cudaError_t rmsnorm_fwd(const void* x, int x_dtype, const float* gamma, float eps, void* n,
                        int n_dtype, float* rstd, float* x_f32_out, int T, int H,
                        cudaStream_t st);
// RMSNorm backward: dx = resid + rstd * gy - x rstd^3 mean(gy x), gy = dy * gamma.
cudaError_t rmsnorm_bwd(const float* dy, const float* x, const float* rstd, const float* gamma,
                        const float* resid, float* dx, int T, int H, cudaStream_t st);

// Encoder head forward: logits = y[b, 0, :] Wh^T + bh; mean CE -> loss; logits_out
// (optional); dlogits [B, C] = (softmax - onehot) / B.
cudaError_t encoder_head_fwd(const void* y, int dtype, const float* Wh, const float* bh,
                             const int32_t* labels, int B, int S, int H, int C, float* loss,
                             float* logits_out, float* dlogits, unsigned* err, cudaStream_t st);
// Encoder head backward: dWh, dbh (nullable), and dy rows at position 0 (dy pre-zeroed).
cudaError_t encoder_head_bwd(const void* y, int dtype, const float* Wh, const float* dlogits,
                             int B, int S, int H, int C, float* dWh, float* dbh, float* dy,
                             cudaStream_t st);
// Span head of extractive QA (start and end logits at every token, Wh [2, H], bh [2]):
// logits_out (optional) [B*S, 2]; dlogits [B*S, 2] = (softmax over the sequence - onehot) /
// (2 B) per column; row_loss [B] = (CE_start + CE_end) / 2; loss = their mean (fixed order).
// labels [B, 2] = (start, end); labels outside [0, S) set RA_DEVERR_BOUNDS and are read as 0.
constexpr int SPAN_MAX_SEQ = 4096;
cudaError_t span_head_fwd(const void* y, int dtype, const float* Wh, const float* bh,
                          const int32_t* labels, int B, int S, int H, float* row_loss, float* loss,
                          float* logits_out, float* dlogits, unsigned* err, cudaStream_t st);
// Its backward: dy [B*S, H] (every row written), and, when dWh / dbh are not null, the head
// gradients through span_head_chunks() token chunks summed in a fixed order; part holds
// span_head_chunks() * (2 H + 2) floats.
int span_head_chunks();
cudaError_t span_head_bwd(const void* y, int dtype, const float* Wh, const float* dlogits, int B,
                          int S, int H, float* dWh, float* dbh, float* dy, float* part,
                          cudaStream_t st);
// Decoder cross-entropy over T rows of V logits (act), in place: logits <- dLoss/dlogits
// (mean over T).  Per-row losses in row_loss, then loss = mean (fixed order).
// Labels outside [0, V) set RA_DEVERR_BOUNDS in *err and are read as 0.
cudaError_t vocab_ce(void* logits, int dtype, int ld, const int32_t* labels, int T, int V,
                     float* row_loss, float* loss, float* logits_out, unsigned* err,
                     cudaStream_t st);

// Adam on a flat fp32 range [0, n): segment s covers [s*seg_len, ...) capped by n; each
// segment has its own step counter steps[s] (incremented by adam_bump).  Also refreshes
// transposed copies through the optional callback-free map below.
struct AdamArgs {
  float* p = nullptr; const float* g = nullptr; float* m = nullptr; float* v = nullptr;
  int64_t n = 0;
  int64_t seg_len = 0;         // elements per segment (one layer's adapters)
  int n_seg = 0;
  const int32_t* steps = nullptr; // [n_seg] completed steps before this update
  float lr = 1e-4f, beta1 = 0.9f, beta2 = 0.999f, eps = 1e-8f;
};
cudaError_t adam_update(const AdamArgs& a, cudaStream_t st);
cudaError_t adam_bump(int32_t* steps, int n, cudaStream_t st);
// Adam over n_layers layers of adapters (a.p / a.g / a.m / a.v at the first layer's start,
// a.steps[l] that layer's completed steps; a.n, a.seg_len and a.n_seg unused) fused with
// the refresh adapter_transpose performs for the same layers.
cudaError_t adam_adapter_update(const AdamArgs& a, float* PT, void* PB, void* PTB, int n_layers,
                                int H, int m, cudaStream_t st);

// Utilities
cudaError_t convert_f32(const float* src, void* dst, int dst_dtype, int64_t n, cudaStream_t st);
// dst[c * ld_dst + r] = src[r, c] (src rows x cols, f32) converted to dst_dtype
cudaError_t transpose_f32(const float* src, void* dst, int dst_dtype, int rows, int cols,
                          int ld_dst, cudaStream_t st);
// Decoder FFN gate/up packing: rows of a part (0 gate, 1 up) [R = F, C = H] go to the packed
// [2F, H] matrix in 64-row blocks alternating gate and up (or to its transpose [H, 2F]).
cudaError_t pack_rows(const float* src, void* dst, int dst_dtype, int R, int C, int part,
                      bool transposed, cudaStream_t st);
// Transposed f32 copies of the adapter matrices of n_layers consecutive layers, and (when
// PB / PTB are given) bf16 copies of both layouts.
cudaError_t adapter_transpose(const float* P, float* PT, void* PB, void* PTB, int n_layers,
                              int H, int m, cudaStream_t st);
cudaError_t fill_f32(float* dst, float v, int64_t n, cudaStream_t st);
// y = f(x) elementwise with the step kernels' own activation code: which 0 GELU, 1 GELU',
// 2 SiLU, 3 SiLU'
cudaError_t eval_activation(int which, const float* x, float* y, int64_t n, cudaStream_t st);

}  // namespace ra
