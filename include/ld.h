/*
 * ld.h -- C ABI of the layer-dropout decoder-stack library (sm_103a).
 *
 * The library runs the forward and backward pass of a pre-norm decoder stack
 * under layer dropout (stochastic depth), as defined in "Don't Drop Dropout"
 * (arXiv 2609.05275):
 *
 *   Eq. (layer_dropout_train), per-sequence case form (Preliminary section):
 *     H^{l+1}[b] = H^l[b]                      with probability p^{l,t}
 *     H^{l+1}[b] = H^l[b] + r f^l(H^l[b])      with probability 1 - p^{l,t}
 *   Eq. (transformer_layer_dropout_train), one mask for both sub-blocks
 *   (layer granularity, Model Granularity subsection):
 *     Z^l = X^l + r M^l f_attn(X^l),   X^{l+1} = Z^l + r M^l f_ffn(Z^l)
 *   or, with sub-layer granularity (same subsection), independent masks
 *   M^l_attn and M^l_ffn in place of M^l in those two updates;
 *   r = alpha / (1 - p) (Dropout Scale paragraph; parameterization table).
 *
 * and, as the Preliminary section's "more efficient implementation" asks, it
 * evaluates f only on the kept sequences: dropped sequences are neither read
 * nor written, in the forward or in the backward.
 *
 * Block: RMSNorm -> fused QKV projection -> RoPE -> causal grouped-query
 * attention -> output projection -> scaled residual; RMSNorm -> SwiGLU
 * gate/up -> down projection -> scaled residual.  No biases, no final norm.
 * The paper's own models (Methodology section) use ALiBi in place of RoPE
 * and a squared-ReLU feed-forward: ld_config.alibi and ld_config.act.
 *
 * Conventions for every entry point
 *   - Device pointers are plain CUDA device addresses owned by the caller;
 *     the library never frees them and keeps none beyond the call, except
 *     that ld_get_masks / ld_sync read the workspace and stream of the last
 *     ld_forward / ld_draw_masks on the handle.
 *   - Matrices are row-major; weights use the [out, in] layout.  The element
 *     type is bf16 (uint16 storage) unless ld_config.fp32_debug is set, in
 *     which case every activation, weight and gain is float32.  Weight and
 *     gain gradients are always float32.
 *   - `stream` is a cudaStream_t (NULL = legacy default stream).  All device
 *     work is ordered on it: ld_backward runs the weight-gradient products
 *     on an internal stream of the handle that forks from `stream` and joins
 *     back into it before the call returns (so the call's work is complete
 *     when `stream` reaches that point, and it can be captured into a CUDA
 *     graph).  No entry point synchronises the host except ld_get_masks and
 *     ld_sync.
 *   - Errors: argument and shape errors are returned synchronously and
 *     enqueue nothing.  A device-side error (a bounded wait that expired) is
 *     recorded in the workspace status word and returned by ld_sync.  No
 *     entry point aborts or throws.
 *   - A handle is not thread-safe; use one per host thread.
 */
#ifndef LD_H
#define LD_H

#include <stddef.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  LD_OK = 0,
  LD_ERR_ARG = 1,      /* null/misaligned pointer, rate outside [0,1], NaN   */
  LD_ERR_SHAPE = 2,    /* unsupported shape (see ld_create)                  */
  LD_ERR_STATE = 3,    /* call out of order (backward without its forward)   */
  LD_ERR_CUDA = 4,     /* a CUDA runtime call failed                         */
  LD_ERR_TIMEOUT = 5,  /* a device-side bounded wait expired                 */
  LD_ERR_OOM = 6,      /* host allocation failed                             */
  LD_ERR_UNSUPPORTED = 7 /* device is not sm_103 / build lacks the kernel    */
} ld_status;

/* Tensor granularity of the masks (Tensor Granularity subsection):
 * per sequence, per batch (one draw per layer and step, shared by every
 * sequence), or per shard: one draw per layer and step for this batch shard
 * alone, keyed by its first global sequence b_offset, so that data-parallel
 * ranks drop different layers while each skips whole layers (the paper's
 * per-device batch dropping; on one device it is the per-batch case).
 * Per token (the finer grain that subsection leaves to future work; this
 * library's reading): one draw per (layer, token); the kept tokens of each
 * sequence run the layer as one shorter sequence in their original order,
 * with rotary angles at their original positions, and a dropped token is
 * left unchanged and contributes no key or value to that layer.  Needs
 * rope_theta or no position scheme (no ALiBi) and, on the bf16 path,
 * Dh = 64 or 128 and S % 128 == 0. */
typedef enum { LD_PER_SEQUENCE = 0, LD_PER_BATCH = 1, LD_PER_SHARD = 2, LD_PER_TOKEN = 3 } ld_granularity;

/* Layer distributions (Dropout Distribution section):
 *   UNIFORM  p^l = p_max
 *   ILD      p^l = l/(L-1) * p_max   (p^0 = 0; a one-layer stack gets 0)
 *   ALD      p^l = p_max * 1[l odd]  (l counted from 0)
 *   EXPLICIT p^l = p_explicit[l]                                          */
typedef enum { LD_DIST_UNIFORM = 0, LD_DIST_ILD = 1, LD_DIST_ALD = 2, LD_DIST_EXPLICIT = 3 } ld_dist;

/* Time schedules (Dropout Schedule section), factor applied to p^l:
 *   CONST 1;  ITS t/(T-1);  DTS 1 - t/(T-1);
 *   RAMP  s0 + (s1-s0) * clamp((t-t0)/(t1-t0), 0, 1)   (warm-up ramp; not
 *         in the paper).  The product is clamped to [0, 1].              */
typedef enum { LD_TIME_CONST = 0, LD_TIME_ITS = 1, LD_TIME_DTS = 2, LD_TIME_RAMP = 3 } ld_time;

/* Feed-forward activation.  SwiGLU: h = silu(g) * u with w_gu = [gate;
 * up] (2F rows).  Squared ReLU (the paper's architecture, Methodology
 * section): h = max(u, 0)^2 with w_gu = up only (F rows). */
typedef enum { LD_ACT_SWIGLU = 0, LD_ACT_RELU2 = 1 } ld_act;

typedef struct {
  int L;            /* layers                                             */
  int d;            /* model width; multiple of 64                        */
  int H, Hkv, Dh;   /* query heads, key/value heads (H % Hkv == 0), head
                       size in {32, 64, 128}; H*Dh multiple of 64          */
  int F;            /* SwiGLU hidden size; multiple of 64                 */
  int B, S;         /* sequences per batch (<= 4096), sequence length
                       (multiple of 64, <= 16384)                         */
  float eps;        /* RMSNorm epsilon, inside the square root            */
  float rope_theta; /* RoPE base; 0 disables the rotary embedding         */
  float alpha;      /* residual multiplier m_L^{-1}; the branch scale is
                       alpha / (1 - p)                                    */
  int granularity;  /* ld_granularity                                     */
  int fp32_debug;   /* 1: float32 storage and SIMT float32 kernels        */
  int b_offset;     /* global index of this batch's sequence 0 (data-
                       parallel shards draw the masks of their global
                       sequences; 0 for an unsharded batch)               */
  int sublayer;     /* 0: one mask per (layer, sequence) for both blocks;
                       1: sub-layer granularity, independent attention and
                       FFN masks, each Bernoulli(1 - p^{l,t})             */
  int alibi;        /* 1: ALiBi position bias, scores of query head h get
                       + m_h (j - i) with the slopes of Press et al. (ICLR
                       2022); requires rope_theta = 0                      */
  int act;          /* ld_act: feed-forward activation                    */
} ld_config;

typedef struct {
  int dist;                  /* ld_dist                                   */
  float p_max;               /* in [0, 1]                                 */
  const float* p_explicit;   /* host, [L], used by LD_DIST_EXPLICIT; copied */
  int time;                  /* ld_time                                   */
  long long T;               /* total steps for ITS / DTS (>= 2)          */
  long long ramp_t0, ramp_t1;/* RAMP window (t1 > t0)                     */
  float ramp_s0, ramp_s1;    /* RAMP factors at t0 and t1                 */
  unsigned long long seed;   /* Philox key                                */
} ld_schedule;

/* Weights of one layer (device pointers, bf16 or float32):
 *   w_qkv [(H+2Hkv)*Dh, d]  rows: Q heads, then K heads, then V heads
 *   w_o   [d, H*Dh]
 *   w_gu  [2F, d]           rows: gate (F), then up (F); [F, d] (up) with
 *                           LD_ACT_RELU2
 *   w_d   [d, F]
 *   g1, g2 [d]              RMSNorm gains before attention / FFN          */
typedef struct { const void *w_qkv, *w_o, *w_gu, *w_d, *g1, *g2; } ld_layer_w;

/* Gradients of one layer (device float32, same shapes; overwritten). */
typedef struct { float *w_qkv, *w_o, *w_gu, *w_d, *g1, *g2; } ld_layer_g;

/* Validate `cfg` and create a handle.  Allocates host memory only (no CUDA
 * call), so it can run without a GPU.  LD_ERR_SHAPE for an unsupported
 * shape, LD_ERR_ARG for null pointers, a non-finite eps/alpha, a flag out of
 * range, ALiBi together with a rotary embedding, or per-token granularity
 * with ALiBi or (bf16 path) with Dh = 32 or S % 128 != 0. */
ld_status ld_create(const ld_config* cfg, void** handle);

/* Bytes of device workspace ld_forward/ld_backward need: the mask tables,
 * the rotary table and, per layer, the activations saved for the backward,
 * sized for the worst case (every sequence kept), plus backward scratch.
 * The caller allocates it (256-byte aligned) and owns it. */
ld_status ld_workspace_size(void* handle, size_t* bytes);

/* Set the drop-rate schedule (host only; the rates of step t are formed at
 * ld_forward / ld_draw_masks time).  LD_ERR_ARG if p_max or an explicit
 * rate is outside [0,1] or NaN, T < 2 for ITS/DTS, or t1 <= t0 for RAMP. */
ld_status ld_set_schedule(void* handle, const ld_schedule* sched);

/* Host-side view of step t: p[l] = p^{l,t} (double), thr[l] =
 * floor(p * 2^32) (the mask drops sequence b iff its Philox word u < thr),
 * scale[l] = alpha / (1 - p) (0 when p = 1).  Any output may be NULL. */
ld_status ld_get_rates(void* handle, long long step, double* p, unsigned long long* thr, float* scale);

/* Draw the masks of step t into the workspace (the first kernel of
 * ld_forward, alone).  Philox4x32-10 (Salmon et al., SC'11): key = (seed
 * low 32 bits, seed high 32 bits), counter = (b', l, t low, t high) with
 * b' = b_offset + b per sequence, b' = 0 per batch and b' = b_offset per
 * shard; word 0 is u (with sub-layer granularity word 0 draws the attention
 * mask and word 1 the FFN mask).  Kept lists are ascending in b (local
 * indices).  Per token: counter (g, l, t low, t high) with g = ((b_offset +
 * b) S + s) mod 2^32, u = word 2 (word 3 for the FFN mask with sub-layer
 * granularity); kept lists hold the rows b S + s, ascending. */
ld_status ld_draw_masks(void* handle, long long step, void* workspace, void* stream);

/* Forward of step t, in place on x [B*S, d] (sequence b = rows b*S..b*S+S-1).
 * W points to L host structs of device pointers.  On the bf16 path the
 * residual stream is carried in a float32 workspace buffer between the
 * layers (x is read once at the start and written once at the end); rows of
 * sequences dropped at every layer come back bit for bit.  Saves what the
 * backward needs in `workspace` and clears the workspace status word. */
ld_status ld_forward(void* handle, long long step, const ld_layer_w* W, void* x, void* workspace,
                     void* stream);

/* Depth-elastic inference forward, Eq. (transformer_layer_dropout_eval):
 *   Z = X + r_eval[l] f_attn(X),  X' = Z + r_eval[l] f_ffn(Z)
 * for every sequence on each layer with execute[l] = 1; layers with
 * execute[l] = 0 are skipped (identity).  Early exit at l' (Inference
 * Optimizations section: run layers 0 .. l'-1) is execute = 1 for l < l',
 * intermediate layer skipping any other pattern.  execute: host [L] of 0/1;
 * r_eval: host [L] or NULL for the paper's r_eval = 1.  x [B*S, d] in place.
 * Needs no schedule and keeps no activations for a backward: `workspace`
 * may be as small as ld_eval_workspace_size (one layer's activations),
 * and a following ld_backward returns LD_ERR_STATE.  The weights of skipped
 * layers are never read (their pointers may be NULL).  LD_ERR_ARG for a
 * null argument, an execute entry other than 0/1, a non-finite r_eval or a
 * missing weight of an executed layer. */
ld_status ld_forward_eval(void* handle, const unsigned char* execute, const float* r_eval, const ld_layer_w* W,
                          void* x, void* workspace, void* stream);

/* Bytes of device workspace ld_forward_eval needs (256-byte aligned). */
ld_status ld_eval_workspace_size(void* handle, size_t* bytes);

/* Backward of the last ld_forward on this handle and workspace (same W).
 * dx [B*S, d] holds dY on entry and dX on return (in place); rows of a
 * sequence dropped at layer l pass through that layer unchanged.  G points
 * to L host structs of device float32 pointers, overwritten with the weight
 * and gain gradients (zero for a layer that kept no sequence).
 * LD_ERR_STATE without a preceding ld_forward on the same workspace. */
ld_status ld_backward(void* handle, const ld_layer_w* W, void* dx, ld_layer_g* G, void* workspace,
                      void* stream);

/* Copy the masks of the last ld_forward / ld_draw_masks to host memory:
 * mask [L*B] (1 = keep), kept_idx [L*B] (ascending, -1 padded), kept_cnt
 * [L]; with sub-layer granularity the attention tables followed by the FFN
 * tables: mask and kept_idx [2*L*B], kept_cnt [2*L].  Per token: mask
 * [L*B*S] (layer l, token b*S+s), kept_idx [L*B*S] (rows b*S+s of the kept
 * tokens, ascending, -1 padded), kept_cnt [L] (kept tokens); [2*L*B*S] and
 * [2*L] with sub-layer granularity.  Synchronises that call's stream.  Any
 * output may be NULL. */
ld_status ld_get_masks(void* handle, unsigned char* mask, int* kept_idx, int* kept_cnt);

/* Synchronise the stream of the last call and return the device status word
 * (LD_OK or LD_ERR_TIMEOUT) accumulated since the last ld_forward /
 * ld_draw_masks on that workspace, clearing it. */
ld_status ld_sync(void* handle);

/* Release the handle (host memory only). */
ld_status ld_destroy(void* handle);

/* Static description of a status code. */
const char* ld_status_str(ld_status status);

/* The CUDA runtime's message for the error behind the last LD_ERR_CUDA that
 * a call of this library returned on the calling thread ("no CUDA error
 * recorded" if none).  The pointer refers to static storage.  Not from the
 * paper: diagnostics of the library. */
const char* ld_last_cuda_error(void);

/* Kernel classes of the device-time accounting below. */
typedef enum {
  LD_KCLASS_GEMM = 0,    /* tcgen05 (or debug SIMT) projections and their gradients */
  LD_KCLASS_ATTN = 1,    /* causal GQA attention, forward and backward              */
  LD_KCLASS_ROWWISE = 2, /* RMSNorm, gathers, RoPE, SwiGLU, reductions              */
  LD_KCLASS_COUNT = 3
} ld_kclass;

/* Device-time accounting (not in the paper; instrumentation for the
 * roofline of each kernel class).  enable = 1 starts recording a CUDA event
 * pair on the call's stream around every launch of ld_forward / ld_backward
 * and resets the totals; enable = 0 stops recording.  The events add no
 * synchronisation.  While recording, ld_backward keeps its weight-gradient
 * products on the caller's stream (no side stream), so that every
 * recorded duration belongs to one launch running alone. */
ld_status ld_set_timing(void* handle, int enable);

/* Sum of the device time (ms) and number of launch groups of class `kclass`
 * recorded since the last ld_set_timing(handle, 1).  Waits for the recorded
 * events to complete. */
ld_status ld_get_timing(void* handle, int kclass, double* ms, long long* launches);

/* Dense contraction used by every projection of the block (the linear maps
 * inside f_attn and f_ffn), exposed for testing and reuse:
 *   D[m, n] = alpha * sum_k A(m, k) * B(n, k),   m < M, n < N, k < K
 * A(m,k) = A[m*lda + k] (a_mn_major = 0) or A[k*lda + m] (a_mn_major = 1);
 * B(n,k) = B[n*ldb + k] (b_mn_major = 0) or B[k*ldb + n] (b_mn_major = 1).
 * A and B are bf16; D is bf16 (d_f32 = 0) or float32 (d_f32 = 1) with row
 * stride ldd.  Runs on the tcgen05 tensor cores with TMA-staged operands.
 * Requirements: M, N, K multiples of 64 (M, N >= 64); lda, ldb, ldd
 * multiples of 8 elements; pointers 16-byte aligned.  Async on `stream`;
 * a device-side timeout sets the status word of `status_ws` (an int on the
 * device, may be NULL). */
ld_status ld_gemm_bf16(int M, int N, int K, const void* A, int lda, int a_mn_major, const void* B,
                       int ldb, int b_mn_major, void* D, int ldd, int d_f32, float alpha,
                       int* status_ws, void* stream);

/* RMSNorm backward with the residual-gradient update on the kept rows of one
 * layer: the last step of each branch of ld_backward (derivative of the
 * pre-norm block of Eq. (transformer_layer_dropout_train) w.r.t. its input
 * through RMSNorm(x) = x / sqrt(mean(x^2) + eps) * gamma).  For compact row
 * m < kept_cnt[0] * S, stored at residual row r = kept_idx[m / S] * S + m % S:
 *   xn = xs[m] * rstd[m],  gd = dyn[m] * gamma
 *   dx[r] += rstd[m] * (gd - xn * mean(gd * xn))            (float32)
 *   next[m] = scale * dx[r]                      (bf16; skipped if NULL)
 *   dgamma  = sum over the kept rows of dyn[m] * xn          (float32)
 * dyn: float [kept*S, d]; xs: float [kept*S, d] (the normalised input's
 * source rows, compact); rstd: float [kept*S]; gamma: bf16 [d]; kept_idx: int [B],
 * kept_cnt: int [1] (device; read by the kernels, so they may be produced
 * on the same stream); dx: float [B*S, d] in/out; dgamma: float [d] out.
 * scratch: float device buffer of scratch_bytes >= nb * d * 4 bytes, nb =
 * min(ceil(B*S / 8), 320), for the per-block partial sums of dgamma.
 * Requires d % 8 == 0, d <= 16384, B, S >= 1; LD_ERR_ARG for null or
 * misaligned pointers or a short scratch buffer.  Async on `stream`. */
ld_status ld_rmsnorm_backward(int B, int S, int d, const float* dyn, const void* xs, const float* rstd,
                              const void* gamma, const int* kept_idx, const int* kept_cnt, float* dx, void* next,
                              float scale, float* dgamma, float* scratch, size_t scratch_bytes, void* stream);

/* The same step as ld_rmsnorm_backward for callers that cannot allocate
 * device memory where they need it (a CUDA graph captured in global mode,
 * where allocation calls are refused during capture; a runtime whose device
 * memory is owned by an allocator this library cannot reach; a path that must
 * not enter an allocator).  The paper has no counterpart: this is a property
 * of the library, not of the method.  Arguments are those of
 * ld_rmsnorm_backward without the scratch buffer: the partial sums of dgamma
 * live in a fixed 10 MiB device array inside the library, which every GPU that
 * loads the library holds until the process exits.  Limit:
 * min(ceil(B*S / 8), 320) * d <= 2,621,440 (e.g. d <= 8192 once B*S >= 2560);
 * larger sizes return LD_ERR_SHAPE.  The first call on each device looks up
 * the array's address with that device current, so make it before any stream
 * capture; the address is kept per device and context, and the first call
 * after cudaDeviceReset (a new context) looks it up again, so that call too
 * belongs before any capture.  All calls share the array: nothing in it needs clearing (each
 * call overwrites every partial sum it reads), but calls that overlap on the
 * GPU race on it and must be serialised by the caller.  Allocates nothing. */
ld_status ld_rmsnorm_backward_noalloc(int B, int S, int d, const float* dyn, const void* xs, const float* rstd,
                                      const void* gamma, const int* kept_idx, const int* kept_cnt, float* dx,
                                      void* next, float scale, float* dgamma, void* stream);

/* Exercise the failure path of the pipelined kernels without a fault: one
 * block waits, with the same bounded wait as every tcgen05 kernel, on an
 * mbarrier phase that nothing completes.  After the wait limit (about 2 s of
 * GPU time) it records LD_ERR_TIMEOUT in *status_ws (an int on the device;
 * a nonzero value already there is kept) and exits; the context stays
 * usable.  Async on `stream`: read *status_ws after synchronising.  The
 * paper has no counterpart: this checks the library's own error handling.
 * LD_ERR_ARG if status_ws is NULL. */
ld_status ld_check_wait_timeout(int* status_ws, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* LD_H */
