/*
 * ringada.h -- C ABI of libringada: the per-batch adapter fine-tuning step of RingAda
 * (arXiv 2502.19864) on one GB300.
 *
 * The step (Algorithm 1, the lines "Perform Fw propagation", "calculates the loss and
 * updates the head", "Perform Bw propagation ending at the (L - d + 1)-th adapter"; and
 * Section III-B.2) is:
 *   ra_forward            forward through all L frozen transformer blocks, each with two
 *                         Houlsby adapters h <- h + GELU(h W_down) W_up (Eq. 1), then the
 *                         head and the mean cross-entropy loss;
 *   ra_backward_truncated the backward from the loss down to the lowest unfrozen layer k
 *                         (0-based, k = L - d), with activation gradients through the
 *                         frozen weights of layers > k and weight gradients only for the
 *                         adapters of layers >= k and the head; layers < k get no work;
 *   ra_adapter_update     Adam on the unfrozen adapters and the trainable head;
 *   ra_set_unfrozen_depth the top-down unfreezing schedule's depth d (Algorithm 1,
 *                         "d = d + 1" every interval; Section III-A).
 *
 * Conventions
 *   - Every pointer named *_dev is a CUDA device pointer; everything else is host memory.
 *   - Device memory is owned by the caller (e.g. PyTorch): the library reports the sizes
 *     it needs (ra_required_bytes) and binds caller buffers (ra_bind_memory).  It never
 *     allocates device memory itself and never frees caller memory.
 *   - Calls that take a cudaStream_t enqueue work on that stream and return; results
 *     land on the device.  Caller inputs must stay valid until the stream reaches the work.
 *     A stream of 0 is the legacy default stream.
 *   - Errors are status codes; nothing throws or aborts.  ra_last_error(ctx) gives a
 *     message for the last failing call on that context.  On error, no work was enqueued
 *     by that call unless stated otherwise.
 *   - Device waits inside kernels are bounded; a wait that runs out records a flag that
 *     ra_sync_status reports as RA_ERR_TIMEOUT.
 *   - Thread safety: one context must not be used from two host threads at once.
 *   - Layout: activations are row-major [B, S, H] (token-major), B*S = T tokens.  Adapter
 *     matrices follow Eq. 1's row-vector convention: W_down [H, m], W_up [m, H].  Frozen
 *     linear weights are [out, in] (the product is x W^T).
 */
#ifndef RINGADA_H
#define RINGADA_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* ra_stream_t; /* same type as cudaStream_t */

typedef enum {
  RA_OK = 0,
  RA_ERR_ARG = 1,         /* a null pointer, out-of-range index or size */
  RA_ERR_STATE = 2,       /* calls out of order (no memory bound, no forward before backward...) */
  RA_ERR_NOT_SAVED = 3,   /* backward asked to reach below the layers the forward saved */
  RA_ERR_SHAPE = 4,       /* B > max_batch, S > max_seq, or an unsupported model shape */
  RA_ERR_NOMEM = 5,       /* a bound buffer is smaller than required */
  RA_ERR_CUDA = 6,        /* a CUDA runtime/driver call failed (message has the CUDA error) */
  RA_ERR_TIMEOUT = 7,     /* a bounded device wait expired (kernel returned early) */
  RA_ERR_UNSUPPORTED = 8  /* no sm_103 device, or a feature this build does not have */
} ra_status;

enum { RA_ENCODER_POSTLN = 0, RA_DECODER_PRENORM = 1, RA_ENCODER_POSTLN_SPAN = 2 };
enum { RA_F32 = 0, RA_BF16 = 1 };
/* Adapter placement (ra_model_cfg.adapter_placement).
 *   RA_ADAPTERS_HOULSBY   two adapters per block, on the attention-output and FFN-output
 *                         branches before their residual add (both archs; parameters
 *                         RA_P_WDA/WUA and RA_P_WDF/WUF);
 *   RA_ADAPTERS_POST_FFN  the placement of the paper's Fig. 1 (Section II-A): one adapter
 *                         per block after the FFN's add & LayerNorm, out = y2 +
 *                         sigma(y2 W_down) W_up (Eq. 1 on the block's LayerNorm output),
 *                         nothing after it; encoders only; its matrices are RA_P_WDF/WUF
 *                         (RA_P_WDA/WUA are not part of such a model).  At the lowest
 *                         unfrozen layer the backward stops right after this adapter's
 *                         weight gradients. */
enum { RA_ADAPTERS_HOULSBY = 0, RA_ADAPTERS_POST_FFN = 1 };

/* Model shape.  Encoder: post-LN blocks (LayerNorm, biased linears, exact-GELU FFN), a
 * trainable n_out-class linear head on the token at position 0.  Span encoder
 * (RA_ENCODER_POSTLN_SPAN): the same blocks with the extractive-QA head of the paper's SQuAD
 * task (Section IV): start and end logits at every token (n_out = 2, max_seq <= 4096), loss
 * = mean over the batch of (CE_start + CE_end) / 2, each a softmax over the sequence.  Decoder: pre-RMSNorm
 * blocks, causal attention with rotate-half RoPE, SwiGLU FFN (ffn % 64 == 0), final
 * RMSNorm and a frozen n_out-way vocabulary head over every position. */
typedef struct {
  int32_t arch;            /* RA_ENCODER_POSTLN | RA_DECODER_PRENORM | RA_ENCODER_POSTLN_SPAN */
  int32_t n_layers;        /* L >= 1 */
  int32_t hidden;          /* H, multiple of 64 */
  int32_t n_heads;         /* H / n_heads in {64, 128} for bf16, <= 128 for f32 */
  int32_t ffn;             /* F, multiple of 64 */
  int32_t n_out;           /* classes (encoder) or vocabulary (decoder), multiple of 8 for decoder bf16 */
  int32_t max_batch;       /* capacity: ra_forward accepts B <= max_batch */
  int32_t max_seq;         /* capacity: ra_forward accepts S <= max_seq */
  int32_t dtype;           /* RA_F32 | RA_BF16: storage of weights and activations */
  int32_t head_trainable;  /* 1: the head is updated with the adapters (encoder); 0: frozen */
  int32_t max_depth;       /* largest unfreezing depth that will be used (0 = L); sizes the
                              saved-activation arena: memory falls as this falls */
  float norm_eps;          /* LayerNorm / RMSNorm epsilon */
  float rope_theta;        /* RoPE base (decoder) */
  int32_t adapter_placement; /* RA_ADAPTERS_HOULSBY (0) | RA_ADAPTERS_POST_FFN (encoders) */
  int32_t prefix_buffers;  /* encoders: 1 reserves the second set of forward scratch buffers
                              and the two prefix outputs of ra_forward_prefix/suffix */
} ra_model_cfg;

typedef struct {
  float lr, beta1, beta2, eps; /* Adam, no weight decay, bias-corrected */
} ra_adam_cfg;

/* Parameter ids for ra_set_weights / ra_get_grad. */
typedef enum {
  /* encoder block */
  RA_P_WQKV = 0, RA_P_BQKV, RA_P_WO, RA_P_BO, RA_P_LN1_G, RA_P_LN1_B,
  RA_P_W1, RA_P_B1, RA_P_W2, RA_P_B2, RA_P_LN2_G, RA_P_LN2_B,
  /* adapters (both archs): attention-branch and FFN-branch, Eq. 1 */
  RA_P_WDA, RA_P_WUA, RA_P_WDF, RA_P_WUF,
  /* decoder block */
  RA_P_WQ, RA_P_WK, RA_P_WV, RA_P_RMS1_G, RA_P_WG, RA_P_WU, RA_P_WD, RA_P_RMS2_G,
  /* head (layer index -1) */
  RA_P_HEAD_W, RA_P_HEAD_B, RA_P_RMSF_G,
  RA_P_COUNT
} ra_param;

typedef struct {
  int32_t layer;       /* 0..L-1, or -1 for the head */
  int32_t param;       /* ra_param */
  const float* data_dev; /* device, float32, row-major in the shape documented for the param;
                            values are rounded once to the model's storage dtype */
  int64_t numel;       /* must equal the param's element count */
} ra_tensor_desc;

typedef struct {
  int64_t weights_bytes, trainable_bytes, workspace_bytes; /* bound sizes */
  int64_t saved_bytes_capacity;  /* arena for max_depth layers */
  int64_t saved_bytes_in_use;    /* activations the last forward kept (layers >= k) */
  int32_t depth;                 /* current unfreezing depth d */
  int32_t k_forward;             /* lowest layer the last forward saved, -1 before any */
  int32_t k_backward;            /* lowest layer the last backward reached, -1 before any */
  int32_t n_updates;             /* completed ra_adapter_update calls */
  int32_t tokens;                /* B*S of the last forward */
  int32_t num_sms;               /* SMs of the bound device */
} ra_stats;

typedef struct ra_ctx ra_ctx;

/* Create a context for the model (host only; no device work).  adapter_dim = m (the
 * bottleneck of Eq. 1), 8 <= m <= 256, multiple of 8.  *out receives the context. */
ra_status ra_create(const ra_model_cfg* cfg, int32_t adapter_dim, ra_ctx** out);

/* Bytes the caller must provide: frozen weights (and their transposed copies),
 * trainable state (adapter/head masters, gradients, Adam moments) and workspace (saved
 * activations for max_depth layers plus scratch).  Each buffer must be 256-byte aligned. */
ra_status ra_required_bytes(const ra_ctx* ctx, size_t* weights, size_t* trainable,
                            size_t* workspace);

/* Bind caller-owned device buffers of at least the required sizes (sizes are given so
 * the library can check them).  Selects the current CUDA device as the context's device;
 * requires compute capability 10.3 (sm_103).  Zeroes gradients, moments and step counts. */
ra_status ra_bind_memory(ra_ctx* ctx, void* weights_dev, size_t weights_bytes,
                         void* trainable_dev, size_t trainable_bytes,
                         void* workspace_dev, size_t workspace_bytes);

/* Copy parameters in (frozen weights, initial adapters and head).  Every parameter of the
 * model must have been set once before the first ra_forward.  Builds the transposed
 * copies the backward reads.  Enqueued on stream. */
ra_status ra_set_weights(ra_ctx* ctx, const ra_tensor_desc* list, int32_t n, ra_stream_t stream);

/* Top-down unfreezing schedule (Algorithm 1: every `interval` rounds the depth grows by
 * one adapter layer, d <- d + 1, from the top down; Section IV unfreezes one more every 40
 * steps): the depth of 0-based step `step` is min(d0 + floor(step / interval), d_max).
 * Host-only, pure.  Returns -1 for step < 0, interval < 1, d0 < 1 or d_max < d0. */
int32_t ra_schedule_depth(int32_t step, int32_t interval, int32_t d0, int32_t d_max);

/* Unfreezing depth d (1..max_depth): the next forward saves activations for layers
 * k = L - d .. L-1 only (Section III-A: below the depth only the forward runs). */
ra_status ra_set_unfrozen_depth(ra_ctx* ctx, int32_t d);

/* Forward and loss (Algorithm 1 "Fw propagation", "calculates the loss").
 * x_dev [B, S, H] in the model dtype; labels_dev int32 [B] (encoder), [B, 2] = (start,
 * end) positions (span encoder) or [B, S] (decoder); loss_dev: one float (mean
 * cross-entropy); logits_dev: nullable, float [B, n_out] (encoder) or [B*S, n_out] (span
 * encoder, decoder).  Returns RA_ERR_SHAPE if B or S exceed capacity.  Labels out of range
 * are read as 0 and reported by ra_sync_status. */
ra_status ra_forward(ra_ctx* ctx, const void* x_dev, const int32_t* labels_dev, int32_t B,
                     int32_t S, float* loss_dev, float* logits_dev, ra_stream_t stream);

/* The same forward split in two, so that the next batch's frozen prefix can run while the
 * current batch is still in its backward and update (Section III-A: the forward below the
 * unfreezing depth is independent of the training above it and can run at the same time;
 * Section III-B.2).  Encoders only; the context needs cfg.prefix_buffers = 1.
 *
 * ra_forward_prefix runs blocks 0 .. k-1 (k = L - d for the depth set now) on x_dev
 * [B, S, H] and leaves the input of block k in prefix buffer `buf` (0 or 1); with k = 0 it
 * copies x_dev there.  It saves nothing and reads only the frozen weights and the adapters
 * of blocks below k, which no update at this or a larger depth writes, and it uses its own
 * scratch buffers: it may run on another stream concurrently with ra_forward_suffix of the
 * other buffer, ra_backward_truncated and ra_adapter_update.  The caller orders it after
 * the ra_forward_suffix that last read the same buffer.
 *
 * ra_forward_suffix runs blocks k .. L-1, the head and the loss from prefix buffer `buf`,
 * with the same arguments and results as ra_forward, and enables the backward as
 * ra_forward does.  The caller orders it after the prefix that filled `buf`.  Returns
 * RA_ERR_STATE if no prefix filled `buf` or the depth changed since, RA_ERR_UNSUPPORTED
 * without prefix buffers (or for a decoder). */
ra_status ra_forward_prefix(ra_ctx* ctx, const void* x_dev, int32_t B, int32_t S, int32_t buf,
                            ra_stream_t stream);
ra_status ra_forward_suffix(ra_ctx* ctx, int32_t buf, const int32_t* labels_dev,
                            float* loss_dev, float* logits_dev, ra_stream_t stream);

/* Backward ending at layer k (0-based; Algorithm 1 "Bw propagation ending at the
 * (L - d + 1)-th adapter" is k = L - d).  Requires a preceding forward; k must satisfy
 * L - d_forward <= k <= L - 1, else RA_ERR_NOT_SAVED (k too low) or RA_ERR_ARG.
 * Writes gradients of the adapters of layers >= k and of the head (if trainable); the
 * gradient buffers of layers < k are not touched.  Gradients are overwritten, not
 * accumulated. */
ra_status ra_backward_truncated(ra_ctx* ctx, int32_t k, ra_stream_t stream);

/* Adam step on the parameters the last backward produced gradients for (adapters of
 * layers >= k_backward, and the head if trainable).  A parameter's step count starts at
 * its first update.  Requires a backward since the last update, else RA_ERR_STATE. */
ra_status ra_adapter_update(ra_ctx* ctx, const ra_adam_cfg* adam, ra_stream_t stream);

/* Device pointer to a float32 gradient buffer (tests): layer 0..L-1 with RA_P_WDA..WUF,
 * or layer -1 with RA_P_HEAD_W / RA_P_HEAD_B.  *n receives the element count.  The
 * pointer stays valid while the memory is bound. */
ra_status ra_get_grad(ra_ctx* ctx, int32_t layer, int32_t which, const float** dev_ptr,
                      int64_t* n);

/* Device pointer to a float32 trainable parameter (master copy), same indexing. */
ra_status ra_get_param(ra_ctx* ctx, int32_t layer, int32_t which, const float** dev_ptr,
                       int64_t* n);

/* Checkpoint of the trainable state: masters, Adam moments, step counts and depth, as an
 * opaque host blob of ra_trainable_state_bytes bytes.  Synchronises the device. */
ra_status ra_trainable_state_bytes(const ra_ctx* ctx, size_t* n);
ra_status ra_get_trainable(ra_ctx* ctx, void* host, size_t n);
ra_status ra_set_trainable(ra_ctx* ctx, const void* host, size_t n);

/* Host-side counters and sizes (no device access). */
ra_status ra_get_stats(const ra_ctx* ctx, ra_stats* out);

/* Synchronise the stream and report whether any bounded wait expired since the last
 * call (RA_ERR_TIMEOUT), or a CUDA error occurred (RA_ERR_CUDA).  Clears the flag. */
ra_status ra_sync_status(ra_ctx* ctx, ra_stream_t stream);

/* Failure-detection hook: enqueues one kernel whose single thread waits, bounded by
 * limit_us microseconds (1 .. 1000000), on a device barrier that nothing ever signals --
 * the same bounded wait every pipelined kernel of the step uses.  The wait expires, the
 * kernel records the timeout and returns; the next ra_sync_status on the stream reports
 * RA_ERR_TIMEOUT and clears it.  Nothing faults or hangs, and the context stays usable. */
ra_status ra_selftest_wait_timeout(ra_ctx* ctx, int32_t limit_us, ra_stream_t stream);

/* Diagnostic: y = f(x) for n float32 values with the activation code the step's kernels
 * use (the sigma of Eq. 1 and its derivative; SiLU of the decoder's SwiGLU FFN).
 * which: 0 GELU(x) = x Phi(x), 1 GELU'(x) = Phi(x) + x phi(x), 2 SiLU, 3 SiLU'.
 * x_dev, y_dev: device arrays of n floats owned by the caller (may alias).  Enqueued on
 * `stream`; RA_ERR_ARG for another `which` or n < 0, RA_ERR_CUDA on a launch error. */
ra_status ra_eval_activation(int32_t which, const float* x_dev, float* y_dev, int64_t n,
                             ra_stream_t stream);

/* Message of the last failing call on ctx (never null; "" if none). */
const char* ra_last_error(const ra_ctx* ctx);

/* Release the context (host memory only; bound device buffers stay the caller's). */
void ra_destroy(ra_ctx* ctx);

/* ---------------------------------------------------------------------------------------
 * Measurement.  With profiling on, every kernel call of the step is bracketed by a pair of
 * CUDA events on the call's stream (also when the calls are captured into a CUDA graph:
 * the events become graph nodes and a replay re-records them).  ra_profile_read sums the
 * elapsed times per category once the recorded work has completed, together with the
 * algorithmic work of those calls (flops: 2 M N K per GEMM, 4 S^2 dh per attention head
 * forward and 10 S^2 dh backward, halved when causal; bytes: each input read once and each
 * output written once).
 * ------------------------------------------------------------------------------------- */
typedef enum {
  RA_PROF_GEMM = 0,     /* frozen-weight GEMMs and their transposed-weight dX GEMMs */
  RA_PROF_ATTN_FWD,     /* fused attention forward */
  RA_PROF_ATTN_BWD,     /* fused attention backward */
  RA_PROF_ADAPTER_FWD,  /* adapter + residual + norm forward */
  RA_PROF_ADAPTER_BWD,  /* adapter backward with the in-kernel dW reduction */
  RA_PROF_NORM,         /* LayerNorm / RMSNorm kernels outside the adapter kernels */
  RA_PROF_HEAD,         /* head, loss, cross-entropy */
  RA_PROF_UPDATE,       /* Adam and the refresh of transposed adapter copies */
  RA_PROF_COUNT
} ra_prof_cat;

typedef struct {
  double ms[RA_PROF_COUNT];     /* summed device time of the calls, milliseconds */
  double flops[RA_PROF_COUNT];  /* algorithmic floating-point operations */
  double bytes[RA_PROF_COUNT];  /* algorithmic DRAM bytes */
  int32_t calls[RA_PROF_COUNT]; /* calls recorded */
} ra_profile;

/* on != 0: start recording (clears earlier records); on == 0: stop recording. */
ra_status ra_profile_enable(ra_ctx* ctx, int32_t on);
/* Sums the records; the caller must have synchronised the recorded work first. */
ra_status ra_profile_read(ra_ctx* ctx, ra_profile* out);
/* The individual records behind ra_profile_read, in call order: category, device
 * milliseconds, algorithmic flops and bytes of each recorded kernel call.  Writes up to
 * `max` records to out (host array) and the total number to *n. */
typedef struct {
  int32_t cat;
  float ms;
  double flops, bytes;
} ra_profile_record;
ra_status ra_profile_records(ra_ctx* ctx, ra_profile_record* out, int32_t max, int32_t* n);
/* Kernels this library has launched in this process so far (every entry point). */
int64_t ra_kernel_launches(void);

/* GEMM timing without per-kernel events (measurement support, no counterpart in the paper).
 * With ra_profile_gemm_log(ctx, 1) every GEMM launch of the following calls (forward,
 * backward) is also recorded: shapes, operands, epilogue and buffers.  ra_profile_gemm_replay
 * enqueues the recorded launches again, in order, back to back on stream (capturable in a
 * CUDA graph), and returns their count and algorithmic flops (2 M N K summed).  Timing that
 * replay gives the GEMM kernels' duration with the launch overlap they have in the step,
 * which an event pair around each kernel removes.  The replay overwrites the step's
 * activations: the next backward needs a new ra_forward (ra_backward_truncated returns
 * RA_ERR_STATE until then). */
ra_status ra_profile_gemm_log(ra_ctx* ctx, int32_t on);
ra_status ra_profile_gemm_replay(ra_ctx* ctx, int32_t* n_launches, double* flops, ra_stream_t stream);

/* ---------------------------------------------------------------------------------------
 * Stand-alone kernels, for testing each piece of the step in isolation.  No context.
 * ------------------------------------------------------------------------------------- */

/* C[M, N] = A[M, K] B[N, K]^T (+ bias[N]) on the tensor cores: bf16 operands, fp32
 * accumulation, bf16 output.  Row-major, leading dimensions equal the row lengths.
 * K % 8 == 0, N % 8 == 0 (16-byte rows).  bias_dev nullable (float).  gelu_out_dev
 * nullable: if given, also writes GELU(C) there (the FFN-up epilogue of the frozen
 * forward).  Returns RA_ERR_UNSUPPORTED on a device that is not sm_103. */
ra_status ra_gemm_bf16(const void* A_dev, const void* B_dev, void* C_dev, int32_t M, int32_t N,
                       int32_t K, const float* bias_dev, void* gelu_out_dev, ra_stream_t stream);

/* The same tensor-core GEMM with one of the step's fused epilogues, for tests and kernel
 * measurements (no counterpart in the paper: these are the step's dense contractions).
 * C = A[M, K] B[N, K]^T accumulated in fp32 (A, B bf16, K-major: lda = ldb = K), then
 *   RA_EPI_STORE       C = acc (+ bias)                  (C bf16 or f32: c_dtype)
 *   RA_EPI_BIAS_GELU   u = acc + bias: C = u (nullable), C2 = GELU(u)     (bf16)
 *   RA_EPI_BIAS_GELU_G u = acc + bias: C = GELU'(u) (nullable), C2 = GELU(u) (bf16)
 *   RA_EPI_MUL         C = acc * aux                     (aux bf16 [M, N], C c_dtype)
 *   RA_EPI_RESID       C = acc + aux                     (aux f32 [M, N], C f32)
 * Outputs are [M, N] row-major with leading dimension N.  bias: nullable f32 [N].  With
 * RA_EPI_B_KN or-ed into epi, B is given as stored [K, N] (N contiguous, leading dimension N),
 * the layout of a forward weight [out, in] that the backward's dX GEMMs multiply by.  Device
 * pointers, 16-byte aligned; N and K multiples of 8.  Enqueued on stream.  RA_ERR_SHAPE
 * for a combination the kernel does not take, RA_ERR_UNSUPPORTED without sm_103.
 * scratch_dev (nullable; 256-byte aligned, scratch_bytes >= ra_gemm_scratch_bytes(),
 * caller-owned, zero-filled before its first use; every call leaves it zeroed): lets the
 * STORE and GELU epilogues spread the k-blocks of a last, partial round of output tiles over
 * all CTAs (stream-K), each such tile summed from its CTAs' fp32 partials in a fixed order,
 * so results are deterministic.  Calls that may run at the same time need different
 * scratch.  Without it every tile is accumulated by one CTA.  RA_ERR_ARG for a scratch
 * that is too small or misaligned. */
enum { RA_EPI_STORE = 0, RA_EPI_BIAS_GELU = 1, RA_EPI_MUL = 2, RA_EPI_RESID = 3,
       RA_EPI_BIAS_GELU_G = 6, RA_EPI_B_KN = 0x100 };
size_t ra_gemm_scratch_bytes(void);
ra_status ra_gemm_bf16_epi(const void* A_dev, const void* B_dev, int32_t M, int32_t N, int32_t K,
                           int32_t epi, const float* bias_dev, const void* aux_dev, void* C_dev,
                           int32_t c_dtype, void* C2_dev, void* scratch_dev, size_t scratch_bytes,
                           ra_stream_t stream);

/* Adapter backward of Eq. 1 for T rows (the in-kernel weight-gradient reduction of the
 * step), float32 throughout.  g_dev [T, H] = dLoss/d(adapter output); h_dev [T, H] the
 * adapter input; z_dev [T, m] = h W_down saved by the forward; W_down [H, m], W_up [m, H].
 * Writes dW_down [H, m], dW_up [m, H] and, if dh_dev is not null, dh [T, H].
 * scratch_dev: caller scratch of ra_adapter_backward_scratch_bytes(T, H, m) bytes.
 * The result is deterministic (fixed reduction order). */
ra_status ra_adapter_backward(const float* g_dev, const float* h_dev, const float* z_dev,
                              const float* W_down_dev, const float* W_up_dev, int32_t T,
                              int32_t H, int32_t m, float* dW_down_dev, float* dW_up_dev,
                              float* dh_dev, void* scratch_dev, size_t scratch_bytes,
                              ra_stream_t stream);
size_t ra_adapter_backward_scratch_bytes(int32_t T, int32_t H, int32_t m);

/* Same computation as ra_adapter_backward, for callers that cannot allocate device memory:
 * plug-in hosts that hand a kernel only its input and output buffers and expose no
 * allocator (custom-operator slots of serving runtimes), and loops that forbid allocation
 * once running, because cudaMalloc can block, synchronise the device or fail at any time.
 * The paper has no counterpart; this is a deployment variant.
 * Scratch: a fixed 16 MiB device array inside the library (ra_adapter_backward_noalloc_
 * capacity() bytes), held on every GPU that loads the library until the process exits;
 * the call allocates nothing and frees nothing.  Sizes whose scratch need
 * (ra_adapter_backward_scratch_bytes) exceeds the array are rejected with RA_ERR_NOMEM.
 * The first call on a device looks up the array's device address (cudaGetSymbolAddress);
 * make that first call before any stream capture.  The address is kept per device together
 * with the CUDA context it belongs to; a call made after that context was destroyed and
 * re-created (e.g. by cudaDeviceReset) looks it up again, so it too should come before any
 * capture.  All calls share the one array: calls
 * that can overlap on the GPU (different streams without ordering) race on it and must be
 * serialised by the caller.  Nothing in the array needs to start at zero: every element a
 * call reads was written earlier in the same call. */
ra_status ra_adapter_backward_noalloc(const float* g_dev, const float* h_dev, const float* z_dev,
                                      const float* W_down_dev, const float* W_up_dev, int32_t T,
                                      int32_t H, int32_t m, float* dW_down_dev, float* dW_up_dev,
                                      float* dh_dev, ra_stream_t stream);
size_t ra_adapter_backward_noalloc_capacity(void);

#ifdef __cplusplus
}
#endif
#endif /* RINGADA_H */
