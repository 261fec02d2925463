// ringada.cu -- C ABI of libringada and the host orchestrator of the step.
//
// One step (Algorithm 1; Section III-B.2):
//   ra_forward            all L blocks forward; blocks below k = L - d keep nothing
//                         (ping-pong scratch), blocks >= k write their saved set into the
//                         arena; then the head and the loss.
//   ra_backward_truncated reverse traversal from the head down to block k, which stops
//                         after its attention-branch adapter's weight gradients.
//   ra_adapter_update     Adam over the suffix [k, L) of adapters plus the head.
#include <cuda.h>
#include <cuda_runtime.h>

#include <atomic>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include "../../include/ringada.h"
#include "kernels.h"

using namespace ra;

namespace {

constexpr size_t kAlign = 256;
// stream-K slots per GEMM scratch set: at least the SM count (one CTA per SM)
constexpr int kSkSlots = 160;
constexpr unsigned RA_DEVERR_TIMEOUT_BIT = 1u;  // matches the device-side flag bits
inline size_t align_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

// Sequential sub-allocator of one caller buffer (offsets first, pointers after binding).
struct Carve {
  size_t off = 0;
  size_t take(size_t bytes) {
    size_t o = off;
    off += align_up(bytes);
    return o;
  }
};

struct LayerWOff {  // offsets into the weights region
  size_t Wqkv, bqkv, Wo, bo, W1, b1, W2, b2, g1, be1, g2, be2;
};
typedef uint16_t bf16_t;  // storage of the bf16 adapter shadows (host side never reads them)

struct SlotOff {  // offsets of one saved-activation slot, relative to the slot base
  // encoder (gp: GELU'(u) of the FFN pre-activation u, saved for the backward)
  size_t qkv, O, lse, a, zA, xhat1, rstd1, gp, f, zF, xhat2, rstd2;
  size_t x_in, x1, gu;                                               // decoder extras
  size_t y2;                                                         // post-FFN adapter input
  size_t full_bytes, lowest_bytes, slot_bytes;
};

}  // namespace

struct ra_ctx {
  ra_model_cfg cfg{};
  int m = 0;
  int L = 0, H = 0, F = 0, nh = 0, dh = 0, C = 0, Tmax = 0, max_depth = 0;
  int act = DT_F32;
  bool dec = false;
  bool span = false;   // encoder with the span (start/end) head over every token
  bool post_ffn = false;  // the paper's placement: one adapter per block after the FFN's add & LN
  std::string err;

  // region sizes and layouts
  size_t w_bytes = 0, t_bytes = 0, ws_bytes = 0;
  std::vector<LayerWOff> lw;
  size_t head_W = 0, head_rmsf = 0;  // decoder frozen head (weights region)
  // trainable region
  size_t n_train = 0;       // floats in P (= G = M = V)
  size_t n_head = 0;        // encoder head floats at the end of P
  size_t t_P = 0, t_G = 0, t_M = 0, t_V = 0, t_PT = 0, t_steps = 0;
  size_t t_PB = 0, t_PTB = 0;  // bf16 shadows of the adapters (both layouts), bf16 models
  // workspace
  SlotOff so{};
  size_t ws_err = 0, ws_arena = 0;
  // GEMM stream-K scratch (bf16 models): flags, then partial slots; set 1 serves the
  // next-batch prefix, which may run on another stream at the same time as set 0
  size_t ws_skf[2]{}, ws_sks[2]{};
  size_t ws_zero_end = 256;  // bytes from the start of the workspace zeroed at binding
  size_t s_X[2]{}, s_qkv = 0, s_O = 0, s_a = 0, s_y1 = 0, s_h = 0, s_f = 0, s_u = 0, s_gu = 0;
  size_t s_n = 0;  // decoder normalised input of the next GEMM
  size_t s_rstd = 0;
  size_t b_dY[2]{}, b_ds2 = 0, b_df = 0, b_du = 0, b_dy1 = 0, b_ds1 = 0, b_da = 0, b_dO = 0,
         b_dqkv = 0, b_dz = 0, b_part = 0, b_D = 0;
  size_t h_dlogits = 0, h_logits = 0, h_rowloss = 0, h_xL = 0, h_nf = 0, h_rstdf = 0;
  size_t h_part = 0;   // span head: token-chunk partials of dWh and dbh

  // bound memory
  char* W = nullptr;
  char* Tr = nullptr;
  char* WS = nullptr;
  int device = -1, num_sms = 0;

  // state
  std::vector<uint8_t> set_mask;  // (L + 1) * RA_P_COUNT
  bool weights_ready = false;
  int depth = 0;
  int k_fwd = -1, k_bwd = -1;
  int fB = 0, fS = 0;
  const int32_t* labels = nullptr;
  bool bwd_since_update = false;
  int n_updates = 0;
  int last_xL_slot = 0;
  const void* yL = nullptr;  // the last block's output of the latest forward (encoder head input)
  // next-batch prefix (ra_forward_prefix / ra_forward_suffix, encoders): a second set of
  // forward scratch buffers, so that the prefix of one batch can run on another stream while
  // the previous batch's suffix, backward and update run, and two buffers for its output
  struct FwdScratch { size_t X[2], qkv, O, a, y1, h, f; int sk; };
  FwdScratch fs[2]{};
  bool prefix_bufs = false;
  size_t pbuf[2]{};
  struct PrefixState { bool valid; int k, B, S; };
  PrefixState pf[2]{};

  // measurement: the GEMM launches of a step, recorded to be replayed back to back
  bool gemm_logging = false;
  std::vector<GemmArgs> gemm_log;
  // profiling: event pairs around kernel calls
  bool profiling = false;
  struct Rec { int cat; double flops, bytes; cudaEvent_t a, b; };
  std::vector<Rec> recs;
  std::vector<cudaEvent_t> pool;
  size_t pool_used = 0;
  cudaEvent_t take_event() {
    if (pool_used == pool.size()) {
      cudaEvent_t e;
      if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
      pool.push_back(e);
    }
    return pool[pool_used++];
  }
  ~ra_ctx() {
    for (cudaEvent_t e : pool) cudaEventDestroy(e);
  }

  template <typename T = void>
  T* w(size_t off) const { return reinterpret_cast<T*>(W + off); }
  template <typename T = void>
  T* ws(size_t off) const { return reinterpret_cast<T*>(WS + off); }
  float* P() const { return reinterpret_cast<float*>(Tr + t_P); }
  float* G() const { return reinterpret_cast<float*>(Tr + t_G); }
  float* PT() const { return reinterpret_cast<float*>(Tr + t_PT); }
  int32_t* steps() const { return reinterpret_cast<int32_t*>(Tr + t_steps); }
  bf16_t* PB() const { return act == DT_BF16 ? reinterpret_cast<bf16_t*>(Tr + t_PB) : nullptr; }
  // bf16 shadow of adapter matrix `mat` (0 WdA [H,m], 1 WuA [m,H], 2 WdF, 3 WuF) of a layer,
  // in the master layout (shadow) or transposed (shadowT); null for fp32 models
  const void* shadow(int layer, int mat) const {
    return act == DT_BF16 ? PB() + (size_t)layer * 4 * H * m + (size_t)mat * H * m : nullptr;
  }
  const void* shadowT(int layer, int mat) const {
    return act == DT_BF16 ? PTB() + (size_t)layer * 4 * H * m + (size_t)mat * H * m : nullptr;
  }
  bf16_t* PTB() const { return act == DT_BF16 ? reinterpret_cast<bf16_t*>(Tr + t_PTB) : nullptr; }
  size_t per_layer_train() const { return (size_t)4 * H * m; }
  char* slot(int layer) const {  // slot base of a saved layer (layer >= L - max_depth)
    int s = layer - (L - max_depth);
    return WS + ws_arena + (size_t)s * so.slot_bytes;
  }
};

namespace {

ra_status fail(ra_ctx* c, ra_status st, const char* fmt, ...) {
  if (c) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    c->err = buf;
  }
  return st;
}

#define CU(expr)                                                                        \
  do {                                                                                  \
    cudaError_t e_ = (expr);                                                            \
    if (e_ != cudaSuccess)                                                              \
      return fail(ctx, RA_ERR_CUDA, "%s failed: %s", #expr, cudaGetErrorString(e_));   \
  } while (0)

int64_t param_numel(const ra_ctx* c, int layer, int p) {
  const int64_t H = c->H, F = c->F, m = c->m, C = c->C;
  if (layer == -1) {
    if (p == RA_P_HEAD_W) return C * H;
    if (p == RA_P_HEAD_B) return c->dec ? -1 : C;
    if (p == RA_P_RMSF_G) return c->dec ? H : -1;
    return -1;
  }
  switch (p) {
    case RA_P_WDA: return c->post_ffn ? -1 : H * m;
    case RA_P_WUA: return c->post_ffn ? -1 : m * H;
    case RA_P_WDF: return H * m;
    case RA_P_WUF: return m * H;
    default: break;
  }
  if (!c->dec) {
    switch (p) {
      case RA_P_WQKV: return 3 * H * H;
      case RA_P_BQKV: return 3 * H;
      case RA_P_WO: return H * H;
      case RA_P_BO: case RA_P_LN1_G: case RA_P_LN1_B: case RA_P_B2: case RA_P_LN2_G:
      case RA_P_LN2_B: return H;
      case RA_P_W1: return F * H;
      case RA_P_B1: return F;
      case RA_P_W2: return H * F;
      default: return -1;
    }
  }
  switch (p) {
    case RA_P_WQ: case RA_P_WK: case RA_P_WV: case RA_P_WO: return H * H;
    case RA_P_RMS1_G: case RA_P_RMS2_G: return H;
    case RA_P_WG: case RA_P_WU: return F * H;
    case RA_P_WD: return H * F;
    default: return -1;
  }
}

void plan(ra_ctx* c) {
  const size_t H = c->H, F = c->F, m = c->m, T = c->Tmax, es = dtype_size(c->act);
  const size_t L = c->L;
  // ---- weights ----
  Carve w;
  c->lw.resize(L);
  for (size_t l = 0; l < L; ++l) {
    LayerWOff& o = c->lw[l];
    o.Wqkv = w.take(3 * H * H * es);
    o.bqkv = c->dec ? 0 : w.take(3 * H * 4);
    o.Wo = w.take(H * H * es);
    o.bo = c->dec ? 0 : w.take(H * 4);
    size_t f1 = c->dec ? 2 * F : F;  // decoder: packed gate|up
    o.W1 = w.take(f1 * H * es);
    o.b1 = c->dec ? 0 : w.take(F * 4);
    o.W2 = w.take(H * F * es);
    o.b2 = c->dec ? 0 : w.take(H * 4);
    o.g1 = w.take(H * 4);
    o.be1 = c->dec ? 0 : w.take(H * 4);
    o.g2 = w.take(H * 4);
    o.be2 = c->dec ? 0 : w.take(H * 4);
  }
  if (c->dec) {
    c->head_W = w.take((size_t)c->C * H * es);
    c->head_rmsf = w.take(H * 4);
  }
  c->w_bytes = w.off;
  // ---- trainable ----
  c->n_head = c->dec ? 0 : (size_t)c->C * H + c->C;  // encoder head lives with the adapters
  c->n_train = L * 4 * H * m + c->n_head;
  Carve t;
  c->t_P = t.take(c->n_train * 4);
  c->t_G = t.take(c->n_train * 4);
  c->t_M = t.take(c->n_train * 4);
  c->t_V = t.take(c->n_train * 4);
  c->t_PT = t.take(L * 4 * H * m * 4);
  c->t_steps = t.take((L + 1) * 4);
  if (c->act == DT_BF16) {
    c->t_PB = t.take(L * 4 * H * m * 2);
    c->t_PTB = t.take(L * 4 * H * m * 2);
  }
  c->t_bytes = t.off;
  // ---- workspace ----
  const size_t Bh = (size_t)c->cfg.max_batch * c->nh * c->cfg.max_seq;  // lse rows
  SlotOff& s = c->so;
  Carve sl;
  // full-only part first (layers > k)
  if (c->dec) s.x_in = sl.take(T * H * 4), s.rstd1 = sl.take(T * 4);
  s.qkv = sl.take(T * 3 * H * es);
  s.O = sl.take(T * H * es);
  s.lse = sl.take(Bh * 4);
  size_t full_only = sl.off;
  if (c->post_ffn) {
    // layers > k: the attention and FFN backward's inputs; layer k: the adapter's alone
    s.xhat1 = sl.take(T * H * es);
    s.rstd1 = sl.take(T * 4);
    s.gp = sl.take(T * F * es);
    s.xhat2 = sl.take(T * H * es);
    s.rstd2 = sl.take(T * 4);
    full_only = sl.off;
    s.y2 = sl.take(T * H * es);
    s.zF = sl.take(T * m * 4);
  } else {
  s.a = sl.take(T * H * es);
  s.zA = sl.take(T * m * 4);
  if (!c->dec) {
    s.xhat1 = sl.take(T * H * es);
    s.rstd1 = sl.take(T * 4);
    s.gp = sl.take(T * F * es);
    s.f = sl.take(T * H * es);
    s.zF = sl.take(T * m * 4);
    s.xhat2 = sl.take(T * H * es);
    s.rstd2 = sl.take(T * 4);
  } else {
    s.x1 = sl.take(T * H * 4);
    s.rstd2 = sl.take(T * 4);
    s.gu = sl.take(T * 2 * F * es);
    s.f = sl.take(T * H * es);
    s.zF = sl.take(T * m * 4);
  }
  }
  s.slot_bytes = sl.off;
  s.full_bytes = sl.off;
  s.lowest_bytes = sl.off - full_only;

  Carve ws;
  c->ws_err = ws.take(256);
  const bool sk = c->act == DT_BF16;
  if (sk) {
    for (int i = 0; i < 2; ++i) c->ws_skf[i] = ws.take((size_t)kSkSlots * gemm_sk_flags_per_slot() * 4);
    c->ws_zero_end = ws.off;
    for (int i = 0; i < 2; ++i) c->ws_sks[i] = ws.take((size_t)kSkSlots * gemm_sk_slot_bytes());
  }
  c->ws_arena = ws.take((size_t)c->max_depth * s.slot_bytes);
  // forward scratch (layers below k)
  if (!c->dec) {
    c->s_X[0] = ws.take(T * H * es);
    c->s_X[1] = ws.take(T * H * es);
  } else {
    c->s_X[0] = ws.take(T * H * 4);
    c->s_X[1] = ws.take(T * H * 4);
    c->s_n = ws.take(T * H * es);
    c->s_rstd = ws.take(T * 4);
  }
  c->s_qkv = ws.take(T * 3 * H * es);
  c->s_O = ws.take(T * H * es);
  c->s_a = ws.take(T * H * es);
  c->s_y1 = ws.take(T * H * (c->dec ? 4 : es));  // decoder: x1 (f32)
  c->s_h = ws.take(T * F * es);
  c->s_f = ws.take(T * H * es);
  c->s_u = c->dec ? 0 : ws.take(T * F * es);
  c->s_gu = c->dec ? ws.take(T * 2 * F * es) : 0;
  c->fs[0] = {{c->s_X[0], c->s_X[1]}, c->s_qkv, c->s_O, c->s_a, c->s_y1, c->s_h, c->s_f, 0};
  c->prefix_bufs = !c->dec && c->cfg.prefix_buffers != 0;
  if (c->prefix_bufs) {
    ra_ctx::FwdScratch& f1 = c->fs[1];
    f1.sk = 1;
    f1.X[0] = ws.take(T * H * es);
    f1.X[1] = ws.take(T * H * es);
    f1.qkv = ws.take(T * 3 * H * es);
    f1.O = ws.take(T * H * es);
    f1.a = ws.take(T * H * es);
    f1.y1 = ws.take(T * H * es);
    f1.h = ws.take(T * F * es);
    f1.f = ws.take(T * H * es);
    c->pbuf[0] = ws.take(T * H * es);
    c->pbuf[1] = ws.take(T * H * es);
  }
  // backward
  c->b_dY[0] = ws.take(T * H * 4);
  c->b_dY[1] = ws.take(T * H * 4);
  c->b_ds2 = ws.take(T * H * 4);
  c->b_df = ws.take(T * H * es);
  c->b_du = ws.take(T * (c->dec ? 2 * F : F) * es);
  c->b_dy1 = ws.take(T * H * 4);
  c->b_ds1 = ws.take(T * H * 4);
  c->b_da = ws.take(T * H * es);
  c->b_dO = ws.take(T * H * es);
  c->b_dqkv = ws.take(T * 3 * H * es);
  c->b_dz = ws.take(T * m * 4);
  c->b_part = ws.take(adapter_bwd_partials_floats(c->Tmax, c->H, c->m) * 4 + 4096);
  c->b_D = ws.take(Bh * 4);
  // head
  c->h_dlogits = ws.take((c->span ? T : (size_t)c->cfg.max_batch) * c->C * 4);
  c->h_rowloss = ws.take(T * 4);
  if (c->span) c->h_part = ws.take((size_t)span_head_chunks() * (2 * H + 2) * 4);
  if (c->dec) {
    c->h_logits = ws.take(T * (size_t)c->C * es);
    c->h_xL = ws.take(T * H * 4);
    c->h_nf = ws.take(T * H * es);
    c->h_rstdf = ws.take(T * 4);
  }
  c->ws_bytes = ws.off;
}

bool is_set(const ra_ctx* c, int layer, int p) {
  return c->set_mask[(size_t)(layer + 1) * RA_P_COUNT + p] != 0;
}

}  // namespace

// =========================================================================================
extern "C" {

ra_status ra_create(const ra_model_cfg* cfg, int32_t adapter_dim, ra_ctx** out) {
  if (!cfg || !out) return RA_ERR_ARG;
  *out = nullptr;
  const ra_model_cfg& g = *cfg;
  if (g.arch != RA_ENCODER_POSTLN && g.arch != RA_DECODER_PRENORM && g.arch != RA_ENCODER_POSTLN_SPAN)
    return RA_ERR_ARG;
  if (g.dtype != RA_F32 && g.dtype != RA_BF16) return RA_ERR_ARG;
  if (g.n_layers < 1 || g.hidden < 64 || g.n_heads < 1 || g.ffn < 1 || g.n_out < 1 ||
      g.max_batch < 1 || g.max_seq < 1)
    return RA_ERR_ARG;
  if (g.max_depth < 0 || g.max_depth > g.n_layers) return RA_ERR_ARG;
  if (adapter_dim < 8 || adapter_dim > 128 || adapter_dim % 8) return RA_ERR_SHAPE;
  if (g.hidden % 64 || g.hidden % g.n_heads || g.ffn % 64) return RA_ERR_SHAPE;
  int dh = g.hidden / g.n_heads;
  if (dh % 32 || dh > 128) return RA_ERR_SHAPE;
  if (g.arch == RA_ENCODER_POSTLN && (g.n_out > 32 || g.max_batch > 256)) return RA_ERR_SHAPE;
  if (g.arch == RA_ENCODER_POSTLN_SPAN && (g.n_out != 2 || g.max_seq > SPAN_MAX_SEQ)) return RA_ERR_SHAPE;
  if (g.arch == RA_DECODER_PRENORM && ((g.dtype == RA_BF16 && g.n_out % 8) || g.head_trainable))
    return RA_ERR_SHAPE;
  if (g.adapter_placement != RA_ADAPTERS_HOULSBY && g.adapter_placement != RA_ADAPTERS_POST_FFN)
    return RA_ERR_ARG;
  if (g.adapter_placement == RA_ADAPTERS_POST_FFN && g.arch == RA_DECODER_PRENORM) return RA_ERR_SHAPE;
  ra_ctx* c = new ra_ctx;
  c->cfg = g;
  c->m = adapter_dim;
  c->L = g.n_layers;
  c->H = g.hidden;
  c->F = g.ffn;
  c->nh = g.n_heads;
  c->dh = dh;
  c->C = g.n_out;
  c->Tmax = g.max_batch * g.max_seq;
  c->max_depth = g.max_depth ? g.max_depth : g.n_layers;
  c->act = g.dtype == RA_BF16 ? DT_BF16 : DT_F32;
  c->dec = g.arch == RA_DECODER_PRENORM;
  c->span = g.arch == RA_ENCODER_POSTLN_SPAN;
  c->post_ffn = g.adapter_placement == RA_ADAPTERS_POST_FFN;
  c->depth = c->max_depth;
  c->set_mask.assign((size_t)(c->L + 1) * RA_P_COUNT, 0);
  plan(c);
  *out = c;
  return RA_OK;
}

ra_status ra_required_bytes(const ra_ctx* c, size_t* weights, size_t* trainable,
                            size_t* workspace) {
  if (!c || !weights || !trainable || !workspace) return RA_ERR_ARG;
  *weights = c->w_bytes;
  *trainable = c->t_bytes;
  *workspace = c->ws_bytes;
  return RA_OK;
}

ra_status ra_bind_memory(ra_ctx* ctx, void* weights_dev, size_t weights_bytes,
                         void* trainable_dev, size_t trainable_bytes, void* workspace_dev,
                         size_t workspace_bytes) {
  if (!ctx) return RA_ERR_ARG;
  if (!weights_dev || !trainable_dev || !workspace_dev)
    return fail(ctx, RA_ERR_ARG, "null buffer");
  if (weights_bytes < ctx->w_bytes || trainable_bytes < ctx->t_bytes ||
      workspace_bytes < ctx->ws_bytes)
    return fail(ctx, RA_ERR_NOMEM, "bound buffers smaller than required");
  if (((uintptr_t)weights_dev | (uintptr_t)trainable_dev | (uintptr_t)workspace_dev) % kAlign)
    return fail(ctx, RA_ERR_ARG, "buffers must be 256-byte aligned");
  int dev = -1;
  CU(cudaGetDevice(&dev));
  cudaDeviceProp prop;
  CU(cudaGetDeviceProperties(&prop, dev));
  if (!(prop.major == 10 && prop.minor == 3))
    return fail(ctx, RA_ERR_UNSUPPORTED, "needs an sm_103 device, found sm_%d%d", prop.major,
                prop.minor);
  ctx->device = dev;
  ctx->num_sms = prop.multiProcessorCount;
  ctx->W = (char*)weights_dev;
  ctx->Tr = (char*)trainable_dev;
  ctx->WS = (char*)workspace_dev;
  CU(cudaMemset(ctx->Tr, 0, ctx->t_bytes));
  CU(cudaMemset(ctx->WS, 0, ctx->ws_zero_end));
  CU(cudaDeviceSynchronize());
  ctx->n_updates = 0;
  ctx->k_fwd = ctx->k_bwd = -1;
  return RA_OK;
}

ra_status ra_set_weights(ra_ctx* ctx, const ra_tensor_desc* list, int32_t n, ra_stream_t stream) {
  if (!ctx) return RA_ERR_ARG;
  if (!ctx->W) return fail(ctx, RA_ERR_STATE, "ra_bind_memory first");
  if (n < 0 || (n > 0 && !list)) return fail(ctx, RA_ERR_ARG, "bad list");
  cudaStream_t st = (cudaStream_t)stream;
  const int H = ctx->H, F = ctx->F, m = ctx->m, act = ctx->act;
  // validate everything before enqueuing anything
  for (int i = 0; i < n; ++i) {
    const ra_tensor_desc& d = list[i];
    if (d.layer < -1 || d.layer >= ctx->L || d.param < 0 || d.param >= RA_P_COUNT || !d.data_dev)
      return fail(ctx, RA_ERR_ARG, "entry %d: bad layer/param/data", i);
    int64_t want = param_numel(ctx, d.layer, d.param);
    if (want < 0) return fail(ctx, RA_ERR_ARG, "entry %d: param %d not in this model", i, d.param);
    if (want != d.numel)
      return fail(ctx, RA_ERR_ARG, "entry %d: numel %lld, expected %lld", i, (long long)d.numel,
                  (long long)want);
  }
  bool adapters_changed = false;
  for (int i = 0; i < n; ++i) {
    const ra_tensor_desc& d = list[i];
    const float* src = d.data_dev;
    const size_t bytes = (size_t)d.numel * 4;
    if (d.layer == -1) {
      if (!ctx->dec) {
        float* dst = ctx->P() + (size_t)ctx->L * 4 * H * m + (d.param == RA_P_HEAD_B ? (size_t)ctx->C * H : 0);
        CU(cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDeviceToDevice, st));
      } else if (d.param == RA_P_HEAD_W) {
        CU(convert_f32(src, ctx->w(ctx->head_W), act, d.numel, st));
      } else {
        CU(cudaMemcpyAsync(ctx->w(ctx->head_rmsf), src, bytes, cudaMemcpyDeviceToDevice, st));
      }
    } else {
      const LayerWOff& o = ctx->lw[d.layer];
      const size_t es = dtype_size(act);
      float* Pl = ctx->P() + (size_t)d.layer * 4 * H * m;
      switch (d.param) {
        case RA_P_WDA: case RA_P_WUA: case RA_P_WDF: case RA_P_WUF: {
          size_t off = (size_t)(d.param - RA_P_WDA) * H * m;
          CU(cudaMemcpyAsync(Pl + off, src, bytes, cudaMemcpyDeviceToDevice, st));
          adapters_changed = true;
        } break;
        case RA_P_WQKV:
          CU(convert_f32(src, ctx->w(o.Wqkv), act, d.numel, st));
          break;
        case RA_P_WQ: case RA_P_WK: case RA_P_WV: {
          int part = d.param - RA_P_WQ;
          CU(convert_f32(src, ctx->w<char>(o.Wqkv) + (size_t)part * H * H * es, act, d.numel, st));
        } break;
        case RA_P_WO:
          CU(convert_f32(src, ctx->w(o.Wo), act, d.numel, st));
          break;
        case RA_P_W1:
          CU(convert_f32(src, ctx->w(o.W1), act, d.numel, st));
          break;
        case RA_P_WG: case RA_P_WU: {
          int part = d.param == RA_P_WU;
          CU(pack_rows(src, ctx->w(o.W1), act, F, H, part, false, st));
        } break;
        case RA_P_W2: case RA_P_WD:
          CU(convert_f32(src, ctx->w(o.W2), act, d.numel, st));
          break;
        case RA_P_BQKV: CU(cudaMemcpyAsync(ctx->w(o.bqkv), src, bytes, cudaMemcpyDeviceToDevice, st)); break;
        case RA_P_BO: CU(cudaMemcpyAsync(ctx->w(o.bo), src, bytes, cudaMemcpyDeviceToDevice, st)); break;
        case RA_P_B1: CU(cudaMemcpyAsync(ctx->w(o.b1), src, bytes, cudaMemcpyDeviceToDevice, st)); break;
        case RA_P_B2: CU(cudaMemcpyAsync(ctx->w(o.b2), src, bytes, cudaMemcpyDeviceToDevice, st)); break;
        case RA_P_LN1_G: case RA_P_RMS1_G: CU(cudaMemcpyAsync(ctx->w(o.g1), src, bytes, cudaMemcpyDeviceToDevice, st)); break;
        case RA_P_LN1_B: CU(cudaMemcpyAsync(ctx->w(o.be1), src, bytes, cudaMemcpyDeviceToDevice, st)); break;
        case RA_P_LN2_G: case RA_P_RMS2_G: CU(cudaMemcpyAsync(ctx->w(o.g2), src, bytes, cudaMemcpyDeviceToDevice, st)); break;
        case RA_P_LN2_B: CU(cudaMemcpyAsync(ctx->w(o.be2), src, bytes, cudaMemcpyDeviceToDevice, st)); break;
        default: return fail(ctx, RA_ERR_ARG, "param %d", d.param);
      }
    }
    ctx->set_mask[(size_t)(d.layer + 1) * RA_P_COUNT + d.param] = 1;
  }
  // transposed and bf16 copies of the adapters the step's kernels read
  if (adapters_changed)
    CU(adapter_transpose(ctx->P(), ctx->PT(), ctx->PB(), ctx->PTB(), ctx->L, H, m, st));
  // every parameter of the model present?
  bool all = true;
  for (int l = -1; l < ctx->L && all; ++l)
    for (int p = 0; p < RA_P_COUNT; ++p)
      if (param_numel(ctx, l, p) > 0 && !is_set(ctx, l, p)) { all = false; break; }
  ctx->weights_ready = all;
  return RA_OK;
}

int32_t ra_schedule_depth(int32_t step, int32_t interval, int32_t d0, int32_t d_max) {
  if (step < 0 || interval < 1 || d0 < 1 || d_max < d0) return -1;
  const int64_t d = (int64_t)d0 + step / interval;
  return (int32_t)(d < d_max ? d : d_max);
}

ra_status ra_set_unfrozen_depth(ra_ctx* ctx, int32_t d) {
  if (!ctx) return RA_ERR_ARG;
  if (d < 1 || d > ctx->max_depth)
    return fail(ctx, RA_ERR_ARG, "depth %d outside 1..%d (max_depth)", d, ctx->max_depth);
  ctx->depth = d;
  return RA_OK;
}

}  // extern "C"

// ---- profiled kernel calls -------------------------------------------------------------
namespace {

template <class F>
cudaError_t prof(ra_ctx* c, int cat, double flops, double bytes, cudaStream_t st, F&& f) {
  if (!c->profiling) return f();
  cudaEvent_t a = c->take_event(), b = c->take_event();
  // inside stream capture an event must be recorded as "external" to become a graph node
  // that a replay re-records (otherwise it only orders the capture)
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  cudaStreamIsCapturing(st, &cs);
  unsigned flags = cs == cudaStreamCaptureStatusActive ? cudaEventRecordExternal : cudaEventRecordDefault;
  if (a) cudaEventRecordWithFlags(a, st, flags);
  cudaError_t e = f();
  if (b) cudaEventRecordWithFlags(b, st, flags);
  if (a && b) c->recs.push_back({cat, flops, bytes, a, b});
  return e;
}

double esz(int dt) { return (double)dtype_size(dt); }

cudaError_t P_gemm(ra_ctx* c, const GemmArgs& g, cudaStream_t st) {
  double M = g.M, N = g.N, K = g.K;
  double out = (g.C ? M * N * esz(g.c_dtype) : 0) + (g.C2 ? M * (g.epi == EPI_SWIGLU ? N / 2 : N) * esz(g.c2_dtype) : 0);
  double aux = g.aux ? M * (g.epi == EPI_DSWIGLU ? 2 * N : N) * esz(g.aux_dtype) : 0;
  if (g.epi == EPI_DSWIGLU) out = 2 * M * N * esz(g.c_dtype);
  double bytes = (M * K + N * K) * esz(g.in_dtype) + out + aux;
  if (c->gemm_logging) c->gemm_log.push_back(g);
  return prof(c, RA_PROF_GEMM, 2 * M * N * K, bytes, st, [&] { return gemm(g, st); });
}

cudaError_t P_attn_fwd(ra_ctx* c, const AttnArgs& a, cudaStream_t st) {
  double S = a.S, bh = (double)a.B * a.n_heads, dh = a.head_dim, T = (double)a.B * a.S;
  double fl = 4 * bh * S * S * dh * (a.causal ? 0.5 : 1.0);
  double by = T * 4 * a.n_heads * dh * esz(a.dtype) + (a.lse ? bh * S * 4 : 0);
  return prof(c, RA_PROF_ATTN_FWD, fl, by, st, [&] { return attention_fwd(a, st); });
}

cudaError_t P_attn_bwd(ra_ctx* c, const AttnArgs& a, cudaStream_t st) {
  double S = a.S, bh = (double)a.B * a.n_heads, dh = a.head_dim, T = (double)a.B * a.S;
  double fl = 10 * bh * S * S * dh * (a.causal ? 0.5 : 1.0);
  double H = (double)a.n_heads * dh;
  double by = T * (3 * H + H + H + 3 * H) * esz(a.dtype) + bh * S * 4;  // qkv, O, dO, dqkv, lse
  return prof(c, RA_PROF_ATTN_BWD, fl, by, st, [&] { return attention_bwd(a, st); });
}

cudaError_t P_adapter_fwd(ra_ctx* c, const AdapterFwdArgs& a, cudaStream_t st) {
  double T = a.T, H = a.H, m = a.m, e = esz(a.dtype);
  double by = T * H * e                              // adapter input
              + T * H * (a.decoder ? 4 : e)          // residual
              + T * H * e                            // normalised output
              + (a.decoder ? T * H * 4 : 0)          // f32 residual stream out
              + (a.xhat ? T * H * e : 0) + (a.rstd ? T * 4 : 0) + (a.z ? T * m * 4 : 0);
  return prof(c, RA_PROF_ADAPTER_FWD, 4 * T * H * m, by, st, [&] { return adapter_fwd(a, st); });
}

cudaError_t P_adapter_bwd(ra_ctx* c, const AdapterBwdArgs& a, cudaStream_t st) {
  double T = a.T, H = a.H, m = a.m, e = esz(a.dtype);
  double by = T * H * 4 + T * H * e + T * m * 4 + (a.dh ? T * H * esz(a.dh_dtype) : 0) + 2 * H * m * 4;
  double fl = 4 * T * H * m + 4 * T * H * m + (a.dh ? 2 * T * H * m : 0);
  return prof(c, RA_PROF_ADAPTER_BWD, fl, by, st, [&] { return adapter_bwd(a, st); });
}

}  // namespace

extern "C" {

// ---- forward -----------------------------------------------------------------------------
namespace {

// sk: the stream-K scratch set (1 for GEMMs of the next-batch prefix, 0 otherwise)
GemmArgs gemm_args(const ra_ctx* c, const void* A, int lda, const void* B, int ldb, int M, int N,
                   int K, int sk = 0) {
  GemmArgs g;
  g.A = A; g.lda = lda; g.B = B; g.ldb = ldb; g.M = M; g.N = N; g.K = K;
  g.in_dtype = c->act;
  g.err = c->ws<unsigned>(c->ws_err);
  if (c->act == DT_BF16) {
    g.sk_ws = c->ws<float>(c->ws_sks[sk]);
    g.sk_flags = c->ws<unsigned>(c->ws_skf[sk]);
    g.sk_slots = kSkSlots;
  }
  return g;
}

// Encoder blocks [l0, l1) on input x with the lowest unfrozen layer k (layers >= k write
// their saved set, layers < k keep nothing).  Scratch comes from the set fs; the block
// outputs ping-pong through fs.X, except that the last block writes last_out when given.
// *y_out receives the last block's output.
// dX GEMMs: C[M, N] = A[M, K] W[K, N] with the forward weight W [out = K, in = N] read as
// stored (row stride ldw), no transposed copy
GemmArgs gemm_kn(const ra_ctx* c, const void* A, int lda, const void* W, int ldw, int M, int N,
                 int K) {
  GemmArgs g = gemm_args(c, A, lda, W, ldw, M, N, K);
  g.b_kn = true;
  return g;
}

ra_status encoder_blocks(ra_ctx* ctx, const void* x, int B, int S, int l0, int l1, int k,
                         const ra_ctx::FwdScratch& fs, void* last_out, const void** y_out,
                         cudaStream_t st) {
  const int H = ctx->H, F = ctx->F, m = ctx->m, T = B * S, act = ctx->act;
  const void* xin = x;
  int out_idx = 0;
  for (int l = l0; l < l1; ++l) {
    const LayerWOff& o = ctx->lw[l];
    const bool saved = l >= k, full = l > k;
    char* sb = saved ? ctx->slot(l) : nullptr;
    const SlotOff& so = ctx->so;
    void* qkv = full ? sb + so.qkv : ctx->ws<char>(fs.qkv);
    void* O = full ? sb + so.O : ctx->ws<char>(fs.O);
    float* lse = full ? (float*)(sb + so.lse) : nullptr;
    void* a = saved ? sb + so.a : ctx->ws<char>(fs.a);
    float* zA = saved ? (float*)(sb + so.zA) : nullptr;
    void* xhat1 = saved ? sb + so.xhat1 : nullptr;
    float* rstd1 = saved ? (float*)(sb + so.rstd1) : nullptr;
    void* gp = saved ? sb + so.gp : nullptr;
    void* f = saved ? sb + so.f : ctx->ws<char>(fs.f);
    float* zF = saved ? (float*)(sb + so.zF) : nullptr;
    void* xhat2 = saved ? sb + so.xhat2 : nullptr;
    float* rstd2 = saved ? (float*)(sb + so.rstd2) : nullptr;
    void* y1 = ctx->ws<char>(fs.y1);
    void* hbuf = ctx->ws<char>(fs.h);
    void* xout = (last_out && l + 1 == l1) ? last_out : ctx->ws<char>(fs.X[out_idx]);
    const float* Pl = ctx->P() + (size_t)l * 4 * H * m;

    GemmArgs g = gemm_args(ctx, xin, H, ctx->w(o.Wqkv), H, T, 3 * H, H, fs.sk);
    g.C = qkv; g.ldc = 3 * H; g.c_dtype = act; g.bias = ctx->w<float>(o.bqkv);
    CU(P_gemm(ctx, g, st));
    AttnArgs at;
    at.qkv = qkv; at.B = B; at.S = S; at.n_heads = ctx->nh; at.head_dim = ctx->dh;
    at.dtype = act; at.scale = 1.f / sqrtf((float)ctx->dh); at.O = O; at.lse = lse;
    at.err = ctx->ws<unsigned>(ctx->ws_err);
    if (!lse) at.lse = nullptr;
    CU(P_attn_fwd(ctx, at, st));
    if (ctx->post_ffn) {
      // Fig. 1 placement: y1 = LN1(x + a); y2 = LN2(y1 + f); out = y2 + GELU(y2 Wd) Wu
      void* a_s = ctx->ws<char>(fs.a);
      g = gemm_args(ctx, O, H, ctx->w(o.Wo), H, T, H, H, fs.sk);
      g.C = a_s; g.ldc = H; g.c_dtype = act; g.bias = ctx->w<float>(o.bo);
      CU(P_gemm(ctx, g, st));
      CU(prof(ctx, RA_PROF_NORM, 0, (double)T * H * ((full ? 4 : 3) * dtype_size(act)), st, [&] {
        return add_layernorm_fwd(xin, a_s, ctx->w<float>(o.g1), ctx->w<float>(o.be1), ctx->cfg.norm_eps,
                                 y1, full ? xhat1 : nullptr, full ? rstd1 : nullptr, T, H, act, st);
      }));
      g = gemm_args(ctx, y1, H, ctx->w(o.W1), H, T, F, H, fs.sk);
      // layers above k keep GELU'(u) for the FFN backward; layer k stops at its adapter
      g.epi = full ? EPI_BIAS_GELU_G : EPI_BIAS_GELU;
      g.C = full ? gp : nullptr; g.ldc = F; g.c_dtype = act; g.bias = ctx->w<float>(o.b1);
      g.C2 = hbuf; g.ldc2 = F; g.c2_dtype = act;
      CU(P_gemm(ctx, g, st));
      void* f_s = ctx->ws<char>(fs.f);
      g = gemm_args(ctx, hbuf, F, ctx->w(o.W2), F, T, H, F, fs.sk);
      g.C = f_s; g.ldc = H; g.c_dtype = act; g.bias = ctx->w<float>(o.b2);
      CU(P_gemm(ctx, g, st));
      // the adapter's input: saved for layers >= k, else scratch (a is consumed by now)
      void* y2 = saved ? sb + so.y2 : a_s;
      CU(prof(ctx, RA_PROF_NORM, 0, (double)T * H * ((full ? 4 : 3) * dtype_size(act)), st, [&] {
        return add_layernorm_fwd(y1, f_s, ctx->w<float>(o.g2), ctx->w<float>(o.be2), ctx->cfg.norm_eps,
                                 y2, full ? xhat2 : nullptr, full ? rstd2 : nullptr, T, H, act, st);
      }));
      AdapterFwdArgs ad;
      ad.T = T; ad.H = H; ad.m = m; ad.dtype = act; ad.no_norm = true;
      ad.a = y2; ad.Wd = Pl + (size_t)2 * H * m; ad.Wu = Pl + (size_t)3 * H * m; ad.z = zF;
      ad.WdT_b = ctx->shadowT(l, 2); ad.WuT_b = ctx->shadowT(l, 3);
      ad.y = xout;
      CU(P_adapter_fwd(ctx, ad, st));
      xin = xout;
      out_idx ^= 1;
      continue;
    }
    g = gemm_args(ctx, O, H, ctx->w(o.Wo), H, T, H, H, fs.sk);
    g.C = a; g.ldc = H; g.c_dtype = act; g.bias = ctx->w<float>(o.bo);
    CU(P_gemm(ctx, g, st));
    AdapterFwdArgs ad;
    ad.T = T; ad.H = H; ad.m = m; ad.dtype = act; ad.decoder = false;
    ad.a = a; ad.Wd = Pl; ad.Wu = Pl + (size_t)H * m; ad.z = zA; ad.resid = xin;
    ad.WdT_b = ctx->shadowT(l, 0); ad.WuT_b = ctx->shadowT(l, 1);
    ad.gamma = ctx->w<float>(o.g1); ad.beta = ctx->w<float>(o.be1); ad.eps = ctx->cfg.norm_eps;
    ad.y = y1; ad.xhat = xhat1; ad.rstd = rstd1;
    CU(P_adapter_fwd(ctx, ad, st));
    g = gemm_args(ctx, y1, H, ctx->w(o.W1), H, T, F, H, fs.sk);
    // saved layers also keep GELU'(u) for the backward; frozen layers need GELU(u) only
    g.epi = gp ? EPI_BIAS_GELU_G : EPI_BIAS_GELU;
    g.C = gp; g.ldc = F; g.c_dtype = act; g.bias = ctx->w<float>(o.b1);
    g.C2 = hbuf; g.ldc2 = F; g.c2_dtype = act;
    CU(P_gemm(ctx, g, st));
    g = gemm_args(ctx, hbuf, F, ctx->w(o.W2), F, T, H, F, fs.sk);
    g.C = f; g.ldc = H; g.c_dtype = act; g.bias = ctx->w<float>(o.b2);
    CU(P_gemm(ctx, g, st));
    ad.a = f; ad.Wd = Pl + (size_t)2 * H * m; ad.Wu = Pl + (size_t)3 * H * m; ad.z = zF;
    ad.WdT_b = ctx->shadowT(l, 2); ad.WuT_b = ctx->shadowT(l, 3);
    ad.resid = y1; ad.gamma = ctx->w<float>(o.g2); ad.beta = ctx->w<float>(o.be2);
    ad.y = xout; ad.xhat = xhat2; ad.rstd = rstd2;
    CU(P_adapter_fwd(ctx, ad, st));
    xin = xout;
    out_idx ^= 1;
  }
  *y_out = xin;
  return RA_OK;
}

// Encoder head and loss on the last block's output y.
ra_status encoder_head_forward(ra_ctx* ctx, const void* xin, int B, int S, float* loss,
                               float* logits, const int32_t* labels, cudaStream_t st) {
  const int L = ctx->L, H = ctx->H, m = ctx->m, T = B * S, act = ctx->act;
  ctx->yL = xin;
  float* Ph = ctx->P() + (size_t)L * 4 * H * m;
  if (ctx->span) {
    // span head: start and end logits at every token of the last block's output
    CU(prof(ctx, RA_PROF_HEAD, 4.0 * T * H, (double)T * H * dtype_size(act), st, [&] {
      return span_head_fwd(xin, act, Ph, Ph + (size_t)2 * H, labels, B, S, H,
                           ctx->ws<float>(ctx->h_rowloss), loss, logits, ctx->ws<float>(ctx->h_dlogits),
                           ctx->ws<unsigned>(ctx->ws_err), st);
    }));
    return RA_OK;
  }
  // head: CLS token of the last block's output
  CU(prof(ctx, RA_PROF_HEAD, 2.0 * B * H * ctx->C, (double)B * H * dtype_size(act), st, [&] {
    return encoder_head_fwd(xin, act, Ph, Ph + (size_t)ctx->C * H, labels, B, S, H, ctx->C, loss,
                            logits, ctx->ws<float>(ctx->h_dlogits), ctx->ws<unsigned>(ctx->ws_err), st);
  }));
  return RA_OK;
}

ra_status encoder_forward(ra_ctx* ctx, const void* x, int B, int S, float* loss, float* logits,
                          const int32_t* labels, cudaStream_t st) {
  const void* y = nullptr;
  ra_status r = encoder_blocks(ctx, x, B, S, 0, ctx->L, ctx->L - ctx->depth, ctx->fs[0], nullptr, &y, st);
  if (r != RA_OK) return r;
  return encoder_head_forward(ctx, y, B, S, loss, logits, labels, st);
}

ra_status decoder_forward(ra_ctx* ctx, const void* x, int B, int S, float* loss, float* logits,
                          const int32_t* labels, cudaStream_t st) {
  const int L = ctx->L, H = ctx->H, F = ctx->F, m = ctx->m, T = B * S, act = ctx->act;
  const int k = ctx->L - ctx->depth;
  const SlotOff& so = ctx->so;
  // layer 0 input: f32 residual stream copy and RMSNorm1
  float* xin = k == 0 ? (float*)(ctx->slot(0) + so.x_in) : ctx->ws<float>(ctx->s_X[0]);
  float* rstd_in = k == 0 ? (float*)(ctx->slot(0) + so.rstd1) : ctx->ws<float>(ctx->s_rstd);
  void* nbuf = ctx->ws<char>(ctx->s_n);
  CU(prof(ctx, RA_PROF_NORM, 0, (double)T * H * (2 * dtype_size(act) + 4), st, [&] {
    return rmsnorm_fwd(x, act, ctx->w<float>(ctx->lw[0].g1), ctx->cfg.norm_eps, nbuf, act, rstd_in,
                       xin, T, H, st);
  }));
  int pp = 1;
  for (int l = 0; l < L; ++l) {
    const LayerWOff& o = ctx->lw[l];
    const bool saved = l >= k, full = l > k;
    char* sb = saved ? ctx->slot(l) : nullptr;
    void* qkv = full ? sb + so.qkv : ctx->ws<char>(ctx->s_qkv);
    void* O = full ? sb + so.O : ctx->ws<char>(ctx->s_O);
    float* lse = full ? (float*)(sb + so.lse) : nullptr;
    void* a = saved ? sb + so.a : ctx->ws<char>(ctx->s_a);
    float* zA = saved ? (float*)(sb + so.zA) : nullptr;
    float* x1 = saved ? (float*)(sb + so.x1) : ctx->ws<float>(ctx->s_y1);
    float* rstd2 = saved ? (float*)(sb + so.rstd2) : ctx->ws<float>(ctx->s_rstd);
    void* gu = saved ? sb + so.gu : ctx->ws<char>(ctx->s_gu);
    void* f = saved ? sb + so.f : ctx->ws<char>(ctx->s_f);
    float* zF = saved ? (float*)(sb + so.zF) : nullptr;
    void* hbuf = ctx->ws<char>(ctx->s_h);
    const float* Pl = ctx->P() + (size_t)l * 4 * H * m;
    // outputs feeding the next layer (or the head)
    float* xnext;
    float* rstd_next;
    const float* gnext;
    if (l + 1 < L) {
      bool next_full = l + 1 > k;
      xnext = next_full ? (float*)(ctx->slot(l + 1) + so.x_in) : ctx->ws<float>(ctx->s_X[pp]);
      rstd_next = next_full ? (float*)(ctx->slot(l + 1) + so.rstd1) : ctx->ws<float>(ctx->s_rstd);
      gnext = ctx->w<float>(ctx->lw[l + 1].g1);
      pp ^= 1;
    } else {
      xnext = ctx->ws<float>(ctx->h_xL);
      rstd_next = ctx->ws<float>(ctx->h_rstdf);
      gnext = ctx->w<float>(ctx->head_rmsf);
    }

    GemmArgs g = gemm_args(ctx, nbuf, H, ctx->w(o.Wqkv), H, T, 3 * H, H);
    g.C = qkv; g.ldc = 3 * H; g.c_dtype = act;
    CU(P_gemm(ctx, g, st));
    AttnArgs at;
    at.qkv = qkv; at.B = B; at.S = S; at.n_heads = ctx->nh; at.head_dim = ctx->dh;
    at.dtype = act; at.causal = true; at.rope = true; at.rope_theta = ctx->cfg.rope_theta;
    at.scale = 1.f / sqrtf((float)ctx->dh); at.O = O; at.lse = lse;
    at.err = ctx->ws<unsigned>(ctx->ws_err);
    if (attention_mma_ok(at)) {
      // q and k rotated once, in place (the saved qkv of this layer then holds them rotated)
      CU(prof(ctx, RA_PROF_ATTN_FWD, 0, (double)T * 2 * H * 2 * esz(act), st,
              [&] { return rope_qk_inplace(at, st); }));
      at.qk_rotated = true;
    }
    CU(P_attn_fwd(ctx, at, st));
    g = gemm_args(ctx, O, H, ctx->w(o.Wo), H, T, H, H);
    g.C = a; g.ldc = H; g.c_dtype = act;
    CU(P_gemm(ctx, g, st));
    AdapterFwdArgs ad;
    ad.T = T; ad.H = H; ad.m = m; ad.dtype = act; ad.decoder = true;
    ad.a = a; ad.Wd = Pl; ad.Wu = Pl + (size_t)H * m; ad.z = zA; ad.resid = xin;
    ad.WdT_b = ctx->shadowT(l, 0); ad.WuT_b = ctx->shadowT(l, 1);
    ad.gamma = ctx->w<float>(o.g2); ad.eps = ctx->cfg.norm_eps;
    ad.y = nbuf; ad.x_out = x1; ad.rstd = rstd2;
    CU(P_adapter_fwd(ctx, ad, st));
    g = gemm_args(ctx, nbuf, H, ctx->w(o.W1), H, T, 2 * F, H);
    g.epi = EPI_SWIGLU; g.C = gu; g.ldc = 2 * F; g.c_dtype = act;
    g.C2 = hbuf; g.ldc2 = F; g.c2_dtype = act;
    CU(P_gemm(ctx, g, st));
    g = gemm_args(ctx, hbuf, F, ctx->w(o.W2), F, T, H, F);
    g.C = f; g.ldc = H; g.c_dtype = act;
    CU(P_gemm(ctx, g, st));
    ad.a = f; ad.Wd = Pl + (size_t)2 * H * m; ad.Wu = Pl + (size_t)3 * H * m; ad.z = zF;
    ad.WdT_b = ctx->shadowT(l, 2); ad.WuT_b = ctx->shadowT(l, 3);
    ad.resid = x1; ad.gamma = gnext;
    ad.y = (l + 1 < L) ? nbuf : ctx->ws<void>(ctx->h_nf);
    ad.x_out = xnext; ad.rstd = rstd_next;
    CU(P_adapter_fwd(ctx, ad, st));
    xin = xnext;
  }
  // head: logits = RMSNorm_f(x_L) Wh^T, CE in place
  void* lg = ctx->ws<char>(ctx->h_logits);
  GemmArgs g = gemm_args(ctx, ctx->ws(ctx->h_nf), H, ctx->w(ctx->head_W), H, T, ctx->C, H);
  g.C = lg; g.ldc = ctx->C; g.c_dtype = act;
  CU(P_gemm(ctx, g, st));
  CU(prof(ctx, RA_PROF_HEAD, 0, 2.0 * T * ctx->C * dtype_size(act), st, [&] {
    return vocab_ce(lg, act, ctx->C, labels, T, ctx->C, ctx->ws<float>(ctx->h_rowloss), loss, logits,
                    ctx->ws<unsigned>(ctx->ws_err), st);
  }));
  return RA_OK;
}

}  // namespace

ra_status ra_forward(ra_ctx* ctx, const void* x_dev, const int32_t* labels_dev, int32_t B,
                     int32_t S, float* loss_dev, float* logits_dev, ra_stream_t stream) {
  if (!ctx) return RA_ERR_ARG;
  if (!ctx->W) return fail(ctx, RA_ERR_STATE, "ra_bind_memory first");
  if (!ctx->weights_ready) return fail(ctx, RA_ERR_STATE, "not every parameter was set");
  if (!x_dev || !labels_dev || !loss_dev) return fail(ctx, RA_ERR_ARG, "null input");
  if (B < 1 || S < 1) return fail(ctx, RA_ERR_ARG, "empty batch");
  if (B > ctx->cfg.max_batch || S > ctx->cfg.max_seq)
    return fail(ctx, RA_ERR_SHAPE, "B=%d S=%d beyond capacity %d x %d", B, S,
                ctx->cfg.max_batch, ctx->cfg.max_seq);
  CU(cudaSetDevice(ctx->device));
  cudaStream_t st = (cudaStream_t)stream;
  ra_status r = ctx->dec ? decoder_forward(ctx, x_dev, B, S, loss_dev, logits_dev, labels_dev, st)
                         : encoder_forward(ctx, x_dev, B, S, loss_dev, logits_dev, labels_dev, st);
  if (r != RA_OK) return r;
  ctx->k_fwd = ctx->L - ctx->depth;
  ctx->fB = B;
  ctx->fS = S;
  ctx->labels = labels_dev;
  ctx->k_bwd = -1;
  return RA_OK;
}

ra_status ra_forward_prefix(ra_ctx* ctx, const void* x_dev, int32_t B, int32_t S, int32_t buf,
                            ra_stream_t stream) {
  if (!ctx) return RA_ERR_ARG;
  if (!ctx->prefix_bufs)
    return fail(ctx, RA_ERR_UNSUPPORTED, "no prefix buffers (encoder with cfg.prefix_buffers = 1)");
  if (!ctx->W) return fail(ctx, RA_ERR_STATE, "ra_bind_memory first");
  if (!ctx->weights_ready) return fail(ctx, RA_ERR_STATE, "not every parameter was set");
  if (!x_dev) return fail(ctx, RA_ERR_ARG, "null input");
  if (buf < 0 || buf > 1) return fail(ctx, RA_ERR_ARG, "buf %d not 0 or 1", buf);
  if (B < 1 || S < 1) return fail(ctx, RA_ERR_ARG, "empty batch");
  if (B > ctx->cfg.max_batch || S > ctx->cfg.max_seq)
    return fail(ctx, RA_ERR_SHAPE, "B=%d S=%d beyond capacity %d x %d", B, S,
                ctx->cfg.max_batch, ctx->cfg.max_seq);
  CU(cudaSetDevice(ctx->device));
  cudaStream_t st = (cudaStream_t)stream;
  const int k = ctx->L - ctx->depth;
  void* out = ctx->ws<char>(ctx->pbuf[buf]);
  ctx->pf[buf].valid = false;
  if (k == 0) {
    CU(cudaMemcpyAsync(out, x_dev, (size_t)B * S * ctx->H * dtype_size(ctx->act),
                       cudaMemcpyDeviceToDevice, st));
  } else {
    const void* y = nullptr;
    ra_status r = encoder_blocks(ctx, x_dev, B, S, 0, k, k, ctx->fs[1], out, &y, st);
    if (r != RA_OK) return r;
  }
  ctx->pf[buf] = {true, k, B, S};
  return RA_OK;
}

ra_status ra_forward_suffix(ra_ctx* ctx, int32_t buf, const int32_t* labels_dev, float* loss_dev,
                            float* logits_dev, ra_stream_t stream) {
  if (!ctx) return RA_ERR_ARG;
  if (!ctx->prefix_bufs)
    return fail(ctx, RA_ERR_UNSUPPORTED, "no prefix buffers (encoder with cfg.prefix_buffers = 1)");
  if (buf < 0 || buf > 1) return fail(ctx, RA_ERR_ARG, "buf %d not 0 or 1", buf);
  if (!labels_dev || !loss_dev) return fail(ctx, RA_ERR_ARG, "null input");
  const int k = ctx->L - ctx->depth;
  const ra_ctx::PrefixState p = ctx->pf[buf];
  if (!p.valid) return fail(ctx, RA_ERR_STATE, "no ra_forward_prefix filled buffer %d", buf);
  if (p.k != k)
    return fail(ctx, RA_ERR_STATE, "the prefix in buffer %d stops at layer %d, the depth now needs %d",
                buf, p.k, k);
  CU(cudaSetDevice(ctx->device));
  cudaStream_t st = (cudaStream_t)stream;
  const void* y = nullptr;
  ra_status r = encoder_blocks(ctx, ctx->ws<char>(ctx->pbuf[buf]), p.B, p.S, k, ctx->L, k, ctx->fs[0],
                               nullptr, &y, st);
  if (r == RA_OK) r = encoder_head_forward(ctx, y, p.B, p.S, loss_dev, logits_dev, labels_dev, st);
  if (r != RA_OK) return r;
  ctx->k_fwd = k;
  ctx->fB = p.B;
  ctx->fS = p.S;
  ctx->labels = labels_dev;
  ctx->k_bwd = -1;
  return RA_OK;
}

// ---- backward ----------------------------------------------------------------------------
ra_status ra_backward_truncated(ra_ctx* ctx, int32_t k, ra_stream_t stream) {
  if (!ctx) return RA_ERR_ARG;
  if (ctx->k_fwd < 0) return fail(ctx, RA_ERR_STATE, "no forward to differentiate");
  if (k > ctx->L - 1 || k < 0) return fail(ctx, RA_ERR_ARG, "k=%d outside 0..L-1", k);
  if (k < ctx->k_fwd)
    return fail(ctx, RA_ERR_NOT_SAVED, "k=%d below the saved depth (forward kept layers >= %d)", k,
                ctx->k_fwd);
  CU(cudaSetDevice(ctx->device));
  cudaStream_t st = (cudaStream_t)stream;
  const int L = ctx->L, H = ctx->H, F = ctx->F, m = ctx->m, act = ctx->act;
  const int B = ctx->fB, S = ctx->fS, T = B * S;
  const SlotOff& so = ctx->so;
  float* dY = ctx->ws<float>(ctx->b_dY[0]);
  int dyi = 0;
  // head
  if (ctx->span) {
    // every token receives a gradient: the span head writes all of dY
    float* Ph = ctx->P() + (size_t)L * 4 * H * m;
    float* Gh = ctx->G() + (size_t)L * 4 * H * m;
    const void* yL = ctx->yL;
    CU(prof(ctx, RA_PROF_HEAD, 8.0 * T * H, (double)T * H * (dtype_size(act) + 4), st, [&] {
      return span_head_bwd(yL, act, Ph, ctx->ws<float>(ctx->h_dlogits), B, S, H,
                           ctx->cfg.head_trainable ? Gh : nullptr,
                           ctx->cfg.head_trainable ? Gh + (size_t)2 * H : nullptr, dY,
                           ctx->ws<float>(ctx->h_part), st);
    }));
  } else if (!ctx->dec) {
    float* Ph = ctx->P() + (size_t)L * 4 * H * m;
    float* Gh = ctx->G() + (size_t)L * 4 * H * m;
    CU(cudaMemsetAsync(dY, 0, (size_t)T * H * 4, st));
    const void* yL = ctx->yL;
    CU(prof(ctx, RA_PROF_HEAD, 4.0 * B * H * ctx->C, (double)B * H * (dtype_size(act) + 4), st, [&] {
      return encoder_head_bwd(yL, act, Ph, ctx->ws<float>(ctx->h_dlogits), B, S, H, ctx->C,
                              ctx->cfg.head_trainable ? Gh : nullptr,
                              ctx->cfg.head_trainable ? Gh + (size_t)ctx->C * H : nullptr, dY, st);
    }));
  } else {
    float* dn = ctx->ws<float>(ctx->b_ds2);
    GemmArgs g = gemm_kn(ctx, ctx->ws(ctx->h_logits), ctx->C, ctx->w(ctx->head_W), H, T,
                           H, ctx->C);
    g.C = dn; g.ldc = H; g.c_dtype = DT_F32;
    CU(P_gemm(ctx, g, st));
    CU(prof(ctx, RA_PROF_NORM, 0, (double)T * H * 12, st, [&] {
      return rmsnorm_bwd(dn, ctx->ws<float>(ctx->h_xL), ctx->ws<float>(ctx->h_rstdf),
                         ctx->w<float>(ctx->head_rmsf), nullptr, dY, T, H, st);
    }));
  }
  // encoder: the layer-output gradient arrives as two parts, dY = (dqkv Wqkv) + ds1 of the
  // layer above; the LayerNorm backward adds them as it loads (null: dY is whole)
  const float* dY2 = nullptr;
  for (int l = L - 1; l >= k; --l) {
    const LayerWOff& o = ctx->lw[l];
    const bool lowest = l == k;
    char* sb = ctx->slot(l);
    const float* PTl = ctx->PT() + (size_t)l * 4 * H * m;
    float* Gl = ctx->G() + (size_t)l * 4 * H * m;
    float* dX = ctx->ws<float>(ctx->b_dY[dyi ^ 1]);
    AdapterBwdArgs ab;
    ab.T = T; ab.H = H; ab.m = m; ab.dtype = act; ab.dz = ctx->ws<float>(ctx->b_dz);
    ab.partials = ctx->ws<float>(ctx->b_part);
    if (ctx->post_ffn) {
      // Fig. 1 placement: the adapter sits on top of the block, so its backward comes first
      // (g = dY, input y2); at layer k the traversal ends right after its weight gradients
      float* dy2 = ctx->ws<float>(ctx->b_ds1);
      ab.g = dY; ab.h = sb + so.y2; ab.z = (float*)(sb + so.zF);
      ab.WuT = PTl + (size_t)3 * H * m; ab.WdT = PTl + (size_t)2 * H * m;
      ab.Wu_b = ctx->shadow(l, 3); ab.Wd_b = ctx->shadow(l, 2);
      ab.dh = lowest ? nullptr : dy2; ab.dh_dtype = DT_F32;
      ab.dWd = Gl + (size_t)2 * H * m; ab.dWu = Gl + (size_t)3 * H * m;
      CU(P_adapter_bwd(ctx, ab, st));
      if (lowest) break;
      // ds2 = LN2'(dy2), kept in f32 for the residual path and in the activation type for
      // the GEMM
      float* ds2 = ctx->ws<float>(ctx->b_ds2);
      CU(prof(ctx, RA_PROF_NORM, 0, (double)T * H * (8 + 2 * dtype_size(act)), st, [&] {
        return layernorm_bwd(dy2, nullptr, sb + so.xhat2, (float*)(sb + so.rstd2), ctx->w<float>(o.g2), ds2,
                             T, H, act, st, ctx->ws(ctx->b_df));
      }));
      GemmArgs g = gemm_kn(ctx, ctx->ws(ctx->b_df), H, ctx->w(o.W2), F, T, F, H);
      g.epi = EPI_MUL; g.C = ctx->ws(ctx->b_du); g.ldc = F; g.c_dtype = act;
      g.aux = sb + so.gp; g.ldaux = F; g.aux_dtype = act;
      CU(P_gemm(ctx, g, st));
      float* dy1 = ctx->ws<float>(ctx->b_dy1);
      g = gemm_kn(ctx, ctx->ws(ctx->b_du), F, ctx->w(o.W1), H, T, H, F);
      g.C = dy1; g.ldc = H; g.c_dtype = DT_F32;
      CU(P_gemm(ctx, g, st));
      float* ds1 = ctx->ws<float>(ctx->b_ds1);
      CU(prof(ctx, RA_PROF_NORM, 0, (double)T * H * (12 + 2 * dtype_size(act)), st, [&] {
        return layernorm_bwd(dy1, ds2, sb + so.xhat1, (float*)(sb + so.rstd1), ctx->w<float>(o.g1), ds1,
                             T, H, act, st, ctx->ws(ctx->b_da));
      }));
      g = gemm_kn(ctx, ctx->ws(ctx->b_da), H, ctx->w(o.Wo), H, T, H, H);
      g.C = ctx->ws(ctx->b_dO); g.ldc = H; g.c_dtype = act;
      CU(P_gemm(ctx, g, st));
      AttnArgs at;
      at.qkv = sb + so.qkv; at.B = B; at.S = S; at.n_heads = ctx->nh; at.head_dim = ctx->dh;
      at.dtype = act; at.scale = 1.f / sqrtf((float)ctx->dh); at.O = sb + so.O;
      at.lse = (float*)(sb + so.lse); at.dO = ctx->ws(ctx->b_dO); at.Dscratch = ctx->ws<float>(ctx->b_D);
      at.dqkv = ctx->ws(ctx->b_dqkv); at.err = ctx->ws<unsigned>(ctx->ws_err);
      CU(P_attn_bwd(ctx, at, st));
      // dX = ds1 + dqkv Wqkv, the residual joined in the GEMM's epilogue (the next layer's
      // adapter backward reads dX whole)
      g = gemm_kn(ctx, ctx->ws(ctx->b_dqkv), 3 * H, ctx->w(o.Wqkv), H, T, H, 3 * H);
      g.epi = EPI_RESID; g.C = dX; g.ldc = H; g.c_dtype = DT_F32;
      g.aux = ds1; g.ldaux = H; g.aux_dtype = DT_F32;
      CU(P_gemm(ctx, g, st));
    } else if (!ctx->dec) {
      float* ds2 = ctx->ws<float>(ctx->b_ds2);
      CU(prof(ctx, RA_PROF_NORM, 0, (double)T * H * (8 + dtype_size(act) + (dY2 ? 4 : 0)), st,
              [&] { return layernorm_bwd(dY, dY2, sb + so.xhat2, (float*)(sb + so.rstd2), ctx->w<float>(o.g2), ds2, T, H, act, st); }));
      // FFN-branch adapter: g = ds2, input f, z_F
      ab.g = ds2; ab.h = sb + so.f; ab.z = (float*)(sb + so.zF);
      ab.WuT = PTl + (size_t)3 * H * m; ab.WdT = PTl + (size_t)2 * H * m;
      ab.Wu_b = ctx->shadow(l, 3); ab.Wd_b = ctx->shadow(l, 2);
      ab.dh = ctx->ws(ctx->b_df); ab.dh_dtype = act;
      ab.dWd = Gl + (size_t)2 * H * m; ab.dWu = Gl + (size_t)3 * H * m;
      CU(P_adapter_bwd(ctx, ab, st));
      // du = (df W2) * GELU'(u), the factor saved by the forward's FFN-up epilogue
      GemmArgs g = gemm_kn(ctx, ctx->ws(ctx->b_df), H, ctx->w(o.W2), F, T, F, H);
      g.epi = EPI_MUL; g.C = ctx->ws(ctx->b_du); g.ldc = F; g.c_dtype = act;
      g.aux = sb + so.gp; g.ldaux = F; g.aux_dtype = act;
      CU(P_gemm(ctx, g, st));
      // dy1 = ds2 + du W1: the GEMM writes du W1, the LayerNorm backward adds ds2
      float* dy1 = ctx->ws<float>(ctx->b_dy1);
      g = gemm_kn(ctx, ctx->ws(ctx->b_du), F, ctx->w(o.W1), H, T, H, F);
      g.C = dy1; g.ldc = H; g.c_dtype = DT_F32;
      CU(P_gemm(ctx, g, st));
      float* ds1 = ctx->ws<float>(ctx->b_ds1);
      CU(prof(ctx, RA_PROF_NORM, 0, (double)T * H * (12 + dtype_size(act)), st,
              [&] { return layernorm_bwd(dy1, ds2, sb + so.xhat1, (float*)(sb + so.rstd1), ctx->w<float>(o.g1), ds1, T, H, act, st); }));
      // attention-branch adapter
      ab.g = ds1; ab.h = sb + so.a; ab.z = (float*)(sb + so.zA);
      ab.WuT = PTl + (size_t)H * m; ab.WdT = PTl;
      ab.Wu_b = ctx->shadow(l, 1); ab.Wd_b = ctx->shadow(l, 0);
      ab.dh = lowest ? nullptr : ctx->ws(ctx->b_da);
      ab.dWd = Gl; ab.dWu = Gl + (size_t)H * m;
      CU(P_adapter_bwd(ctx, ab, st));
      if (lowest) break;
      g = gemm_kn(ctx, ctx->ws(ctx->b_da), H, ctx->w(o.Wo), H, T, H, H);
      g.C = ctx->ws(ctx->b_dO); g.ldc = H; g.c_dtype = act;
      CU(P_gemm(ctx, g, st));
      AttnArgs at;
      at.qkv = sb + so.qkv; at.B = B; at.S = S; at.n_heads = ctx->nh; at.head_dim = ctx->dh;
      at.dtype = act; at.scale = 1.f / sqrtf((float)ctx->dh); at.O = sb + so.O;
      at.lse = (float*)(sb + so.lse); at.dO = ctx->ws(ctx->b_dO); at.Dscratch = ctx->ws<float>(ctx->b_D);
      at.dqkv = ctx->ws(ctx->b_dqkv); at.err = ctx->ws<unsigned>(ctx->ws_err);
      CU(P_attn_bwd(ctx, at, st));
      // dX = ds1 + dqkv Wqkv: the GEMM writes dqkv Wqkv; the next layer's LayerNorm backward
      // adds ds1
      g = gemm_kn(ctx, ctx->ws(ctx->b_dqkv), 3 * H, ctx->w(o.Wqkv), H, T, H, 3 * H);
      g.C = dX; g.ldc = H; g.c_dtype = DT_F32;
      CU(P_gemm(ctx, g, st));
      dY2 = ds1;
    } else {
      // FFN-branch adapter: g = dY (= d x2), input f, z_F
      ab.g = dY; ab.h = sb + so.f; ab.z = (float*)(sb + so.zF);
      ab.WuT = PTl + (size_t)3 * H * m; ab.WdT = PTl + (size_t)2 * H * m;
      ab.Wu_b = ctx->shadow(l, 3); ab.Wd_b = ctx->shadow(l, 2);
      ab.dh = ctx->ws(ctx->b_df); ab.dh_dtype = act;
      ab.dWd = Gl + (size_t)2 * H * m; ab.dWu = Gl + (size_t)3 * H * m;
      CU(P_adapter_bwd(ctx, ab, st));
      // d(gate), d(up) from d h = df Wd
      GemmArgs g = gemm_kn(ctx, ctx->ws(ctx->b_df), H, ctx->w(o.W2), F, T, F, H);
      g.epi = EPI_DSWIGLU; g.C = ctx->ws(ctx->b_du); g.ldc = 2 * F; g.c_dtype = act;
      g.aux = sb + so.gu; g.ldaux = 2 * F; g.aux_dtype = act;
      CU(P_gemm(ctx, g, st));
      float* dn2 = ctx->ws<float>(ctx->b_ds2);
      g = gemm_kn(ctx, ctx->ws(ctx->b_du), 2 * F, ctx->w(o.W1), H, T, H, 2 * F);
      g.C = dn2; g.ldc = H; g.c_dtype = DT_F32;
      CU(P_gemm(ctx, g, st));
      float* dx1 = ctx->ws<float>(ctx->b_dy1);
      CU(prof(ctx, RA_PROF_NORM, 0, (double)T * H * 16, st,
              [&] { return rmsnorm_bwd(dn2, (float*)(sb + so.x1), (float*)(sb + so.rstd2), ctx->w<float>(o.g2), dY, dx1, T, H, st); }));
      ab.g = dx1; ab.h = sb + so.a; ab.z = (float*)(sb + so.zA);
      ab.WuT = PTl + (size_t)H * m; ab.WdT = PTl;
      ab.Wu_b = ctx->shadow(l, 1); ab.Wd_b = ctx->shadow(l, 0);
      ab.dh = lowest ? nullptr : ctx->ws(ctx->b_da);
      ab.dWd = Gl; ab.dWu = Gl + (size_t)H * m;
      CU(P_adapter_bwd(ctx, ab, st));
      if (lowest) break;
      g = gemm_kn(ctx, ctx->ws(ctx->b_da), H, ctx->w(o.Wo), H, T, H, H);
      g.C = ctx->ws(ctx->b_dO); g.ldc = H; g.c_dtype = act;
      CU(P_gemm(ctx, g, st));
      AttnArgs at;
      at.qkv = sb + so.qkv; at.B = B; at.S = S; at.n_heads = ctx->nh; at.head_dim = ctx->dh;
      at.dtype = act; at.causal = true; at.rope = true; at.rope_theta = ctx->cfg.rope_theta;
      at.qk_rotated = attention_mma_ok(at);  // the forward rotated the saved q and k in place
      at.scale = 1.f / sqrtf((float)ctx->dh); at.O = sb + so.O;
      at.lse = (float*)(sb + so.lse); at.dO = ctx->ws(ctx->b_dO); at.Dscratch = ctx->ws<float>(ctx->b_D);
      at.dqkv = ctx->ws(ctx->b_dqkv); at.err = ctx->ws<unsigned>(ctx->ws_err);
      CU(P_attn_bwd(ctx, at, st));
      float* dn1 = ctx->ws<float>(ctx->b_ds1);
      g = gemm_kn(ctx, ctx->ws(ctx->b_dqkv), 3 * H, ctx->w(o.Wqkv), H, T, H, 3 * H);
      g.C = dn1; g.ldc = H; g.c_dtype = DT_F32;
      CU(P_gemm(ctx, g, st));
      CU(prof(ctx, RA_PROF_NORM, 0, (double)T * H * 16, st,
              [&] { return rmsnorm_bwd(dn1, (float*)(sb + so.x_in), (float*)(sb + so.rstd1), ctx->w<float>(o.g1), dx1, dX, T, H, st); }));
    }
    dY = dX;
    dyi ^= 1;
  }
  ctx->k_bwd = k;
  ctx->bwd_since_update = true;
  return RA_OK;
}

// ---- update ------------------------------------------------------------------------------
ra_status ra_adapter_update(ra_ctx* ctx, const ra_adam_cfg* adam, ra_stream_t stream) {
  if (!ctx || !adam) return RA_ERR_ARG;
  if (!ctx->bwd_since_update || ctx->k_bwd < 0)
    return fail(ctx, RA_ERR_STATE, "no backward since the last update");
  if (!(adam->lr >= 0.f) || !(adam->beta1 >= 0.f && adam->beta1 < 1.f) ||
      !(adam->beta2 >= 0.f && adam->beta2 < 1.f) || !(adam->eps > 0.f))
    return fail(ctx, RA_ERR_ARG, "bad Adam hyper-parameters");
  CU(cudaSetDevice(ctx->device));
  cudaStream_t st = (cudaStream_t)stream;
  const int L = ctx->L, k = ctx->k_bwd;
  const size_t per = ctx->per_layer_train();
  const size_t off = (size_t)k * per;
  AdamArgs a;
  a.p = ctx->P() + off;
  a.g = ctx->G() + off;
  a.m = reinterpret_cast<float*>(ctx->Tr + ctx->t_M) + off;
  a.v = reinterpret_cast<float*>(ctx->Tr + ctx->t_V) + off;
  a.n = (int64_t)(ctx->n_train - off - (ctx->cfg.head_trainable ? 0 : ctx->n_head));
  a.seg_len = (int64_t)per;
  a.n_seg = (L - k) + (ctx->cfg.head_trainable ? 1 : 0);
  a.steps = ctx->steps() + k;
  a.lr = adam->lr; a.beta1 = adam->beta1; a.beta2 = adam->beta2; a.eps = adam->eps;
  // adapters: Adam fused with the transposed / bf16 refresh; the encoder head (when trained)
  // is one more segment through the plain kernel; the step counters advance last
  AdamArgs h = a;
  h.p = a.p + (size_t)(L - k) * per;
  h.g = a.g + (size_t)(L - k) * per;
  h.m = a.m + (size_t)(L - k) * per;
  h.v = a.v + (size_t)(L - k) * per;
  h.n = a.n - (int64_t)((L - k) * per);
  h.seg_len = h.n > 0 ? h.n : 1;
  h.n_seg = 1;
  h.steps = a.steps + (L - k);
  const size_t adapt = (size_t)(L - k) * per;
  // per adapter element: g, m, v, p read and m, v, p written (28 B), PT (4 B), PB + PTB (4 B)
  const double bytes = (double)adapt * (ctx->PB() ? 36 : 32) + (double)(h.n > 0 ? h.n : 0) * 28;
  CU(prof(ctx, RA_PROF_UPDATE, 0, bytes, st, [&] {
    cudaError_t e = adam_adapter_update(a, ctx->PT() + off, ctx->PB() ? ctx->PB() + off : nullptr,
                                        ctx->PTB() ? ctx->PTB() + off : nullptr, L - k, ctx->H, ctx->m, st);
    if (e == cudaSuccess && h.n > 0) e = adam_update(h, st);
    if (e == cudaSuccess) e = adam_bump(ctx->steps() + k, a.n_seg, st);
    return e;
  }));
  ctx->bwd_since_update = false;
  ctx->n_updates++;
  return RA_OK;
}

// ---- inspection ----------------------------------------------------------------------------
namespace {
ra_status locate(ra_ctx* ctx, int32_t layer, int32_t which, float* base, const float** p,
                 int64_t* n) {
  if (!ctx->Tr) return fail(ctx, RA_ERR_STATE, "ra_bind_memory first");
  const size_t H = ctx->H, m = ctx->m;
  if (layer >= 0 && layer < ctx->L && which >= RA_P_WDA && which <= RA_P_WUF &&
      !(ctx->post_ffn && (which == RA_P_WDA || which == RA_P_WUA))) {
    *p = base + (size_t)layer * 4 * H * m + (size_t)(which - RA_P_WDA) * H * m;
    *n = (int64_t)(H * m);
    return RA_OK;
  }
  if (layer == -1 && !ctx->dec && (which == RA_P_HEAD_W || which == RA_P_HEAD_B)) {
    *p = base + (size_t)ctx->L * 4 * H * m + (which == RA_P_HEAD_B ? (size_t)ctx->C * H : 0);
    *n = which == RA_P_HEAD_W ? (int64_t)ctx->C * H : ctx->C;
    return RA_OK;
  }
  return fail(ctx, RA_ERR_ARG, "no trainable tensor at layer %d param %d", layer, which);
}
}  // namespace

ra_status ra_get_grad(ra_ctx* ctx, int32_t layer, int32_t which, const float** dev_ptr, int64_t* n) {
  if (!ctx || !dev_ptr || !n) return RA_ERR_ARG;
  return locate(ctx, layer, which, ctx->Tr ? ctx->G() : nullptr, dev_ptr, n);
}

ra_status ra_get_param(ra_ctx* ctx, int32_t layer, int32_t which, const float** dev_ptr, int64_t* n) {
  if (!ctx || !dev_ptr || !n) return RA_ERR_ARG;
  return locate(ctx, layer, which, ctx->Tr ? ctx->P() : nullptr, dev_ptr, n);
}

// checkpoint blob: [magic, version, n_train, L, depth, n_updates] int64 header, then P, M, V
// (float), then steps (int32, L + 1)
namespace {
constexpr int64_t kMagic = 0x52696e6741646131LL;  // "RingAda1"
size_t blob_bytes(const ra_ctx* c) {
  return 6 * sizeof(int64_t) + 3 * c->n_train * sizeof(float) + (size_t)(c->L + 1) * sizeof(int32_t);
}
}  // namespace

ra_status ra_trainable_state_bytes(const ra_ctx* ctx, size_t* n) {
  if (!ctx || !n) return RA_ERR_ARG;
  *n = blob_bytes(ctx);
  return RA_OK;
}

ra_status ra_get_trainable(ra_ctx* ctx, void* host, size_t n) {
  if (!ctx || !host) return RA_ERR_ARG;
  if (!ctx->Tr) return fail(ctx, RA_ERR_STATE, "ra_bind_memory first");
  if (n != blob_bytes(ctx)) return fail(ctx, RA_ERR_ARG, "blob size %zu, expected %zu", n, blob_bytes(ctx));
  CU(cudaSetDevice(ctx->device));
  CU(cudaDeviceSynchronize());
  int64_t* hdr = (int64_t*)host;
  hdr[0] = kMagic; hdr[1] = 1; hdr[2] = (int64_t)ctx->n_train; hdr[3] = ctx->L;
  hdr[4] = ctx->depth; hdr[5] = ctx->n_updates;
  char* p = (char*)host + 6 * sizeof(int64_t);
  const size_t fb = ctx->n_train * sizeof(float);
  CU(cudaMemcpy(p, ctx->Tr + ctx->t_P, fb, cudaMemcpyDeviceToHost));
  CU(cudaMemcpy(p + fb, ctx->Tr + ctx->t_M, fb, cudaMemcpyDeviceToHost));
  CU(cudaMemcpy(p + 2 * fb, ctx->Tr + ctx->t_V, fb, cudaMemcpyDeviceToHost));
  CU(cudaMemcpy(p + 3 * fb, ctx->Tr + ctx->t_steps, (ctx->L + 1) * sizeof(int32_t), cudaMemcpyDeviceToHost));
  return RA_OK;
}

ra_status ra_set_trainable(ra_ctx* ctx, const void* host, size_t n) {
  if (!ctx || !host) return RA_ERR_ARG;
  if (!ctx->Tr) return fail(ctx, RA_ERR_STATE, "ra_bind_memory first");
  if (n != blob_bytes(ctx)) return fail(ctx, RA_ERR_ARG, "blob size %zu, expected %zu", n, blob_bytes(ctx));
  const int64_t* hdr = (const int64_t*)host;
  if (hdr[0] != kMagic || hdr[1] != 1 || hdr[2] != (int64_t)ctx->n_train || hdr[3] != ctx->L)
    return fail(ctx, RA_ERR_ARG, "checkpoint does not match this model");
  if (hdr[4] < 1 || hdr[4] > ctx->max_depth) return fail(ctx, RA_ERR_ARG, "checkpoint depth out of range");
  CU(cudaSetDevice(ctx->device));
  CU(cudaDeviceSynchronize());
  const char* p = (const char*)host + 6 * sizeof(int64_t);
  const size_t fb = ctx->n_train * sizeof(float);
  CU(cudaMemcpy(ctx->Tr + ctx->t_P, p, fb, cudaMemcpyHostToDevice));
  CU(cudaMemcpy(ctx->Tr + ctx->t_M, p + fb, fb, cudaMemcpyHostToDevice));
  CU(cudaMemcpy(ctx->Tr + ctx->t_V, p + 2 * fb, fb, cudaMemcpyHostToDevice));
  CU(cudaMemcpy(ctx->Tr + ctx->t_steps, p + 3 * fb, (ctx->L + 1) * sizeof(int32_t), cudaMemcpyHostToDevice));
  CU(adapter_transpose(ctx->P(), ctx->PT(), ctx->PB(), ctx->PTB(), ctx->L, ctx->H, ctx->m, 0));
  CU(cudaDeviceSynchronize());
  ctx->depth = (int)hdr[4];
  ctx->n_updates = (int)hdr[5];
  ctx->k_fwd = ctx->k_bwd = -1;
  ctx->bwd_since_update = false;
  return RA_OK;
}

ra_status ra_get_stats(const ra_ctx* ctx, ra_stats* out) {
  if (!ctx || !out) return RA_ERR_ARG;
  ra_stats s{};
  s.weights_bytes = (int64_t)ctx->w_bytes;
  s.trainable_bytes = (int64_t)ctx->t_bytes;
  s.workspace_bytes = (int64_t)ctx->ws_bytes;
  s.saved_bytes_capacity = (int64_t)ctx->max_depth * (int64_t)ctx->so.slot_bytes;
  if (ctx->k_fwd >= 0) {
    int d = ctx->L - ctx->k_fwd;
    s.saved_bytes_in_use = (int64_t)(d - 1) * (int64_t)ctx->so.full_bytes + (int64_t)ctx->so.lowest_bytes;
  }
  s.depth = ctx->depth;
  s.k_forward = ctx->k_fwd;
  s.k_backward = ctx->k_bwd;
  s.n_updates = ctx->n_updates;
  s.tokens = ctx->fB * ctx->fS;
  s.num_sms = ctx->num_sms;
  *out = s;
  return RA_OK;
}

ra_status ra_sync_status(ra_ctx* ctx, ra_stream_t stream) {
  if (!ctx) return RA_ERR_ARG;
  if (!ctx->WS) return fail(ctx, RA_ERR_STATE, "ra_bind_memory first");
  CU(cudaSetDevice(ctx->device));
  CU(cudaStreamSynchronize((cudaStream_t)stream));
  CU(cudaGetLastError());
  unsigned flag = 0;
  CU(cudaMemcpy(&flag, ctx->WS + ctx->ws_err, sizeof flag, cudaMemcpyDeviceToHost));
  if (flag) {
    CU(cudaMemset(ctx->WS + ctx->ws_err, 0, sizeof flag));
    if (flag & RA_DEVERR_TIMEOUT_BIT)
      return fail(ctx, RA_ERR_TIMEOUT, "a bounded device wait expired (flags 0x%x)", flag);
    return fail(ctx, RA_ERR_ARG, "a device input was out of range, e.g. a label (flags 0x%x)", flag);
  }
  return RA_OK;
}

ra_status ra_selftest_wait_timeout(ra_ctx* ctx, int32_t limit_us, ra_stream_t stream) {
  if (!ctx) return RA_ERR_ARG;
  if (!ctx->WS) return fail(ctx, RA_ERR_STATE, "ra_bind_memory first");
  if (limit_us < 1 || limit_us > 1000000) return fail(ctx, RA_ERR_ARG, "limit_us outside 1..1000000");
  CU(cudaSetDevice(ctx->device));
  CU(selftest_wait(ctx->ws<unsigned>(ctx->ws_err), (uint64_t)limit_us * 1000ull, (cudaStream_t)stream));
  return RA_OK;
}

ra_status ra_eval_activation(int32_t which, const float* x_dev, float* y_dev, int64_t n,
                             ra_stream_t stream) {
  if (which < 0 || which > 3 || n < 0 || (n > 0 && (!x_dev || !y_dev))) return RA_ERR_ARG;
  return eval_activation(which, x_dev, y_dev, n, (cudaStream_t)stream) == cudaSuccess ? RA_OK : RA_ERR_CUDA;
}

const char* ra_last_error(const ra_ctx* ctx) { return ctx ? ctx->err.c_str() : "null context"; }

void ra_destroy(ra_ctx* ctx) { delete ctx; }

// ---- measurement -------------------------------------------------------------------------
ra_status ra_profile_enable(ra_ctx* ctx, int32_t on) {
  if (!ctx) return RA_ERR_ARG;
  ctx->profiling = on != 0;
  if (on) {
    ctx->recs.clear();
    ctx->pool_used = 0;
  }
  return RA_OK;
}

ra_status ra_profile_read(ra_ctx* ctx, ra_profile* out) {
  if (!ctx || !out) return RA_ERR_ARG;
  ra_profile p{};
  for (const auto& r : ctx->recs) {
    float ms = 0.f;
    cudaError_t e = cudaEventElapsedTime(&ms, r.a, r.b);
    if (e != cudaSuccess) return fail(ctx, RA_ERR_CUDA, "cudaEventElapsedTime: %s", cudaGetErrorString(e));
    p.ms[r.cat] += ms;
    p.flops[r.cat] += r.flops;
    p.bytes[r.cat] += r.bytes;
    p.calls[r.cat] += 1;
  }
  *out = p;
  return RA_OK;
}

ra_status ra_profile_records(ra_ctx* ctx, ra_profile_record* out, int32_t max, int32_t* n) {
  if (!ctx || !n || (max > 0 && !out)) return RA_ERR_ARG;
  int32_t i = 0;
  for (const auto& r : ctx->recs) {
    if (i < max) {
      float ms = 0.f;
      cudaError_t e = cudaEventElapsedTime(&ms, r.a, r.b);
      if (e != cudaSuccess) return fail(ctx, RA_ERR_CUDA, "cudaEventElapsedTime: %s", cudaGetErrorString(e));
      out[i] = ra_profile_record{r.cat, ms, r.flops, r.bytes};
    }
    ++i;
  }
  *n = i;
  return RA_OK;
}

int64_t ra_kernel_launches(void) { return (int64_t)launches_so_far(); }

ra_status ra_profile_gemm_log(ra_ctx* ctx, int32_t on) {
  if (!ctx) return RA_ERR_ARG;
  ctx->gemm_logging = on != 0;
  if (on) ctx->gemm_log.clear();
  return RA_OK;
}

ra_status ra_profile_gemm_replay(ra_ctx* ctx, int32_t* n_launches, double* flops, ra_stream_t stream) {
  if (!ctx) return RA_ERR_ARG;
  if (!ctx->W) return fail(ctx, RA_ERR_STATE, "ra_bind_memory first");
  CU(cudaSetDevice(ctx->device));
  double fl = 0.0;
  for (const GemmArgs& g : ctx->gemm_log) {
    CU(gemm(g, (cudaStream_t)stream));
    fl += 2.0 * g.M * g.N * g.K;
  }
  if (n_launches) *n_launches = (int32_t)ctx->gemm_log.size();
  if (flops) *flops = fl;
  ctx->k_fwd = ctx->k_bwd = -1;  // the replay overwrote the saved activations
  ctx->bwd_since_update = false;
  return RA_OK;
}

// ---- stand-alone kernels -----------------------------------------------------------------
ra_status ra_gemm_bf16(const void* A_dev, const void* B_dev, void* C_dev, int32_t M, int32_t N,
                       int32_t K, const float* bias_dev, void* gelu_out_dev, ra_stream_t stream) {
  if (!A_dev || !B_dev || !C_dev || M < 0 || N <= 0 || K <= 0) return RA_ERR_ARG;
  if (K % 8 || N % 8) return RA_ERR_SHAPE;
  if (!tc_available()) return RA_ERR_UNSUPPORTED;
  GemmArgs g;
  g.A = A_dev; g.lda = K; g.B = B_dev; g.ldb = K; g.M = M; g.N = N; g.K = K;
  g.in_dtype = DT_BF16;
  g.C = C_dev; g.ldc = N; g.c_dtype = DT_BF16; g.bias = bias_dev;
  if (gelu_out_dev) { g.epi = EPI_BIAS_GELU; g.C2 = gelu_out_dev; g.ldc2 = N; g.c2_dtype = DT_BF16; }
  cudaError_t e = gemm_tc(g, (cudaStream_t)stream);
  if (e == cudaErrorNotSupported) return RA_ERR_SHAPE;
  return e == cudaSuccess ? RA_OK : RA_ERR_CUDA;
}

size_t ra_gemm_scratch_bytes(void) {
  return align_up((size_t)kSkSlots * gemm_sk_flags_per_slot() * 4) + (size_t)kSkSlots * gemm_sk_slot_bytes();
}

ra_status ra_gemm_bf16_epi(const void* A_dev, const void* B_dev, int32_t M, int32_t N, int32_t K,
                           int32_t epi, const float* bias_dev, const void* aux_dev, void* C_dev,
                           int32_t c_dtype, void* C2_dev, void* scratch_dev, size_t scratch_bytes,
                           ra_stream_t stream) {
  if (!A_dev || !B_dev || M < 0 || N <= 0 || K <= 0) return RA_ERR_ARG;
  if (scratch_dev && (scratch_bytes < ra_gemm_scratch_bytes() || (uintptr_t)scratch_dev % kAlign))
    return RA_ERR_ARG;
  if (c_dtype != RA_F32 && c_dtype != RA_BF16) return RA_ERR_ARG;
  if (K % 8 || N % 8) return RA_ERR_SHAPE;
  const bool b_kn = (epi & RA_EPI_B_KN) != 0;
  epi &= ~RA_EPI_B_KN;
  GemmArgs g;
  g.A = A_dev; g.lda = K; g.B = B_dev; g.ldb = b_kn ? N : K; g.b_kn = b_kn;
  g.M = M; g.N = N; g.K = K;
  g.in_dtype = DT_BF16;
  g.C = C_dev; g.ldc = N; g.c_dtype = c_dtype == RA_BF16 ? DT_BF16 : DT_F32;
  switch (epi) {
    case RA_EPI_STORE:
      if (!C_dev) return RA_ERR_ARG;
      g.epi = EPI_STORE; g.bias = bias_dev;
      break;
    case RA_EPI_BIAS_GELU:
    case RA_EPI_BIAS_GELU_G:
      if (!C2_dev || c_dtype != RA_BF16) return RA_ERR_ARG;
      g.epi = epi == RA_EPI_BIAS_GELU ? EPI_BIAS_GELU : EPI_BIAS_GELU_G;
      g.bias = bias_dev; g.C2 = C2_dev; g.ldc2 = N; g.c2_dtype = DT_BF16;
      break;
    case RA_EPI_MUL:
      if (!C_dev || !aux_dev) return RA_ERR_ARG;
      g.epi = EPI_MUL; g.aux = aux_dev; g.ldaux = N; g.aux_dtype = DT_BF16;
      break;
    case RA_EPI_RESID:
      if (!C_dev || !aux_dev || c_dtype != RA_F32) return RA_ERR_ARG;
      g.epi = EPI_RESID; g.aux = aux_dev; g.ldaux = N; g.aux_dtype = DT_F32;
      break;
    default: return RA_ERR_ARG;
  }
  if (scratch_dev) {
    g.sk_flags = (unsigned*)scratch_dev;
    g.sk_ws = (float*)((char*)scratch_dev + align_up((size_t)kSkSlots * gemm_sk_flags_per_slot() * 4));
    g.sk_slots = kSkSlots;
  }
  if (!tc_available()) return RA_ERR_UNSUPPORTED;
  cudaError_t e = gemm_tc(g, (cudaStream_t)stream);
  if (e == cudaErrorNotSupported) return RA_ERR_SHAPE;
  return e == cudaSuccess ? RA_OK : RA_ERR_CUDA;
}

size_t ra_adapter_backward_scratch_bytes(int32_t T, int32_t H, int32_t m) {
  if (T < 1 || H < 1 || m < 1) return 0;
  return adapter_bwd_partials_floats(T, H, m) * 4 + (size_t)T * m * 4 + 2 * (size_t)H * m * 4 + 3 * kAlign;
}

ra_status ra_adapter_backward(const float* g_dev, const float* h_dev, const float* z_dev,
                              const float* W_down_dev, const float* W_up_dev, int32_t T,
                              int32_t H, int32_t m, float* dW_down_dev, float* dW_up_dev,
                              float* dh_dev, void* scratch_dev, size_t scratch_bytes,
                              ra_stream_t stream) {
  if (!g_dev || !h_dev || !z_dev || !W_down_dev || !W_up_dev || !dW_down_dev || !dW_up_dev || !scratch_dev)
    return RA_ERR_ARG;
  if (T < 1 || H < 1 || m < 1) return RA_ERR_ARG;
  if (m > 128) return RA_ERR_SHAPE;
  if (scratch_bytes < ra_adapter_backward_scratch_bytes(T, H, m)) return RA_ERR_NOMEM;
  cudaStream_t st = (cudaStream_t)stream;
  char* s = (char*)scratch_dev;
  Carve cv;
  float* part = (float*)(s + cv.take(adapter_bwd_partials_floats(T, H, m) * 4));
  float* dz = (float*)(s + cv.take((size_t)T * m * 4));
  float* WuT = (float*)(s + cv.take((size_t)H * m * 4));
  float* WdT = (float*)(s + cv.take((size_t)H * m * 4));
  if (transpose_f32(W_up_dev, WuT, DT_F32, m, H, m, st) != cudaSuccess) return RA_ERR_CUDA;
  if (transpose_f32(W_down_dev, WdT, DT_F32, H, m, H, st) != cudaSuccess) return RA_ERR_CUDA;
  AdapterBwdArgs a;
  a.T = T; a.H = H; a.m = m; a.dtype = DT_F32;
  a.g = g_dev; a.h = h_dev; a.z = z_dev; a.WuT = WuT; a.WdT = WdT; a.dz = dz;
  a.dh = dh_dev; a.dh_dtype = DT_F32; a.dWd = dW_down_dev; a.dWu = dW_up_dev; a.partials = part;
  return adapter_bwd(a, st) == cudaSuccess ? RA_OK : RA_ERR_CUDA;
}

}  // extern "C"

namespace ra {
static std::atomic<long long> g_launches{0};
void note_launch(int n) { g_launches.fetch_add(n, std::memory_order_relaxed); }
long long launches_so_far() { return g_launches.load(std::memory_order_relaxed); }

int device_sm_count() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 148;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) return 148;
  return n;
}
}  // namespace ra
