// Internal declarations shared by the translation units of the library.
// Not part of the C ABI (include/ld.h is).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/ld.h"

#define LD_MAX_L 256
#define LD_MAX_B 4096

namespace ldk {

// Element storage: bf16 on the tensor-core path, float on the debug path.
typedef __nv_bfloat16 bf16;

__device__ __forceinline__ float to_f(float v) { return v; }
__device__ __forceinline__ float to_f(bf16 v) { return __bfloat162float(v); }
template <typename T> __device__ __forceinline__ T from_f(float v);
template <> __device__ __forceinline__ float from_f<float>(float v) { return v; }
template <> __device__ __forceinline__ bf16 from_f<bf16>(float v) { return __float2bfloat16_rn(v); }

// Device status word: 0 = ok, LD_ERR_TIMEOUT when a bounded wait expired.
__device__ __forceinline__ void set_status(int* status, int code) {
  if (status) atomicCAS(status, 0, code);
}

// Nanosecond wall clock of the GPU (for bounded waits).
__device__ __forceinline__ uint64_t gtimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Every spin-wait in the library gives up after this long and reports
// LD_ERR_TIMEOUT through the status word.
constexpr uint64_t kWaitLimitNs = 2000000000ull;

// Row of the residual stream for compact row m of layer l: sequence
// kept_idx[m / S], position m % S.  Per-token kept lists are passed with
// S = 1 (kept_idx[m] is then the token's row b S + s); their padding rows
// hold -1, so the result is negative for them and callers skip the row.
__device__ __forceinline__ long long src_row(const int* kept_idx, int S, long long m) {
  const long long k = kept_idx[m / S];
  return k < 0 ? -1 : k * S + (m % S);
}

// Position of compact row m in its sequence: m % S when the compact rows
// are whole kept sequences of S rows (tok = null), else tok[m] % S with tok
// the per-token kept list (rows b S + s; padding rows -1 get position 0).
__device__ __forceinline__ int row_pos(const int* tok, int S, long long m) {
  if (!tok) return (int)(m % S);
  const int t = tok[m];
  return t < 0 ? 0 : t % S;
}

// ------------------------------------------------------------------------
// launchers (host side); each returns cudaGetLastError()
// ------------------------------------------------------------------------

struct MaskParams {
  unsigned long long seed;
  long long step;
  int L, B, S, granularity, b_offset;
  int nmask;  // 1: one mask per (layer, sequence); 2: attention (word 0) and FFN (word 1) masks
  unsigned long long thr[LD_MAX_L];
};
// Per sequence / batch / shard: mask [nmask][L][B], kept_idx [nmask][L][B]
// (kept sequences ascending, -1 after), kept_cnt [nmask][L] (sequences).
// Per token: mask [nmask][L][B*S], kept_idx [nmask][L][B*S] (rows b S + s of
// the kept tokens ascending, then -1), kept_cnt [nmask][L] = the kept-token
// count rounded up to a multiple of 64 (the row extent of the layer's
// products; the padding rows hold -1), seg [nmask][L][B+1] (the kept tokens
// of sequence b are compact rows seg[b] .. seg[b+1]-1; seg[B] = the count).
cudaError_t launch_mask_compact(const MaskParams& P, unsigned char* mask, int* kept_idx, int* kept_cnt, int* seg,
                                cudaStream_t st);

// Zero rows [*start, min(*start + nrows, max_rows)) of `planes` row-major
// matrices (plane p at buf + p * plane_ld elements, row stride ld, the first
// ncols columns), one element per thread.
template <typename T>
cudaError_t launch_zero_rows(T* buf, int ld, int ncols, int planes, long long plane_ld, const int* start, int nrows,
                             int max_rows, cudaStream_t st);

// Elementwise copy with conversion between float32 and bf16 (n % 8 == 0).
cudaError_t launch_convert(const void* src, int src_f32, void* dst, int dst_f32, long long n, cudaStream_t st);

cudaError_t launch_rope_table(float* cos_t, float* sin_t, int S, int Dh, double theta, cudaStream_t st);

// ALiBi slopes m_h of H heads (natural units) into slopes[H].
cudaError_t launch_alibi_table(float* slopes, int H, cudaStream_t st);

// RMSNorm forward over the rows of layer l (M = *cnt * S rows).  When
// `gather` is set the source row of compact row m is src_row(kept_idx, S, m)
// of the float32 residual stream, else row m of a compact buffer.  Writes
// the normalised rows (out), the reciprocal rms (rstd) and, if copy != null,
// a compact copy of the source rows.
template <typename TS, typename T>
cudaError_t launch_rmsnorm_fwd(const TS* src, int gather, const int* kept_idx, const int* cnt, int S, int d,
                               int max_rows, const T* gamma, float eps, TS* copy, T* out, float* rstd,
                               cudaStream_t st);

// RMSNorm backward + residual: for compact row m with source row r,
//   dx[r] += rstd (dyn*g - xn * mean(dyn*g*xn)),  xn = xs[m] * rstd[m]
// on the float32 residual gradient dx (dyn is float32), then, if next != null,
// next[m] = scale * dx[r] (compact, for the next branch).  Partial gain
// gradients go to part[blockIdx][d] (nblocks blocks, a launch constant).
template <typename T>
cudaError_t launch_rmsnorm_bwd(const float* dyn, const float* xs, const float* rstd, const T* gamma, float* dx,
                               const int* kept_idx, const int* cnt, int S, int d, int max_rows, float scale,
                               T* next, float* part, int nblocks, cudaStream_t st);
int rmsnorm_bwd_blocks(int max_rows);
cudaError_t launch_colsum(const float* part, int nrows, int d, float* out, cudaStream_t st);

// out[m] = scale * dx[src_row(m)] from the float32 residual gradient.
template <typename T>
cudaError_t launch_gather_scale(const float* dx, const int* kept_idx, const int* cnt, int S, int d, int max_rows,
                                float scale, T* out, cudaStream_t st);

// Rows: (*cnt) * S compact rows at positions m % S, or, with tok (per-token
// kept list), *cnt rows at positions tok[m] % S.
template <typename T>
cudaError_t launch_rope_apply(T* qkv, int ld, int nheads, int Dh, const float* cos_t, const float* sin_t,
                              const int* cnt, int S, int max_rows, int inverse, const int* tok, cudaStream_t st);

template <typename T>
cudaError_t launch_swiglu_fwd(const T* gu, T* h, const int* cnt, int S, int F, int max_rows, cudaStream_t st);

template <typename T>
cudaError_t launch_swiglu_bwd(const T* dh, const T* gu, T* dgu, const int* cnt, int S, int F, int max_rows,
                              cudaStream_t st);

// Squared ReLU over [M, F] rows: out = max(u, 0)^2 if dh is null, else
// out = dh * 2 max(u, 0).
template <typename T>
cudaError_t launch_relu2(const T* u, const T* dh, T* out, const int* cnt, int S, int F, int max_rows,
                         cudaStream_t st);

template <typename T>
cudaError_t launch_attn_rowdot(const T* dO, const T* O, int ld, int H, int Dh, const int* cnt, int S, int max_rows,
                               float* Dvec, cudaStream_t st);

// Every attention launcher takes `alibi`: null, or the device table of the
// H ALiBi slopes (scores of head h get + m_h (j - i)), and `seg`, `tok`:
// null for whole kept sequences (*cnt of them, S rows each), or the
// per-token segments (sequence b = compact rows seg[b] .. seg[b+1]-1, b <
// max_seqs) and kept list (position tok[m] % S; -1 rows belong to no
// sequence).  Per-token attention takes no ALiBi table.
// Reference (SIMT) attention, used by the float32 debug path.
template <typename T>
cudaError_t launch_attn_fwd_simt(const T* qkv, int ldqkv, T* o, int ldo, float* lse, const int* cnt, int S, int H,
                                 int Hkv, int Dh, int max_rows, const float* alibi, const int* seg, const int* tok,
                                 cudaStream_t st);
template <typename T>
cudaError_t launch_attn_bwd_simt(const T* qkv, int ldqkv, const T* dO, int ldo, const float* lse, const float* Dvec,
                                 T* dqkv, const int* cnt, int S, int H, int Hkv, int Dh, int max_rows,
                                 const float* alibi, const int* seg, const int* tok, cudaStream_t st);

// Tensor-core (mma.sync) flash attention for bf16.
cudaError_t launch_attn_fwd_mma(const bf16* qkv, int ldqkv, bf16* o, int ldo, float* lse, const int* cnt, int S,
                                int H, int Hkv, int Dh, int max_seqs, const float* alibi, cudaStream_t st);
cudaError_t launch_attn_bwd_mma(const bf16* qkv, int ldqkv, const bf16* o, const bf16* dO, int ldo,
                                const float* lse, const float* Dvec, float* dq_acc, bf16* dqkv, const int* cnt,
                                int S, int H, int Hkv, int Dh, int max_seqs, const float* alibi, cudaStream_t st);
// tcgen05 flash attention forward (head size 64 or 128, S % 128 == 0).
bool attn_tc_supported(int S, int Dh);
cudaError_t launch_attn_fwd_tc(const bf16* qkv, int ldqkv, bf16* o, int ldo, float* lse, const int* cnt, int S, int H,
                               int Hkv, int Dh, int max_seqs, const float* alibi, const int* seg, int* status,
                               cudaStream_t st);
// tcgen05 flash attention backward (head sizes 64 and 128, S % 128 == 0):
// dQ (scaled by 1/sqrt(Dh)), dK and dV into dqkv, dQ and dK with the inverse
// RoPE applied (rcos = null: no rotation).  Head size 128 accumulates dQ in
// dq_acc (zeroed here) and finishes it with launch_dq_finish; head size 64
// does not touch dq_acc.
bool attn_bwd_tc_supported(int S, int Dh);
cudaError_t launch_attn_bwd_tc(const bf16* qkv, int ldqkv, const bf16* dO, int ldo, const float* lse,
                               const float* Dvec, float* dq_acc, bf16* dqkv, const int* cnt, int S, int H, int Hkv,
                               int Dh, int max_seqs, const float* rcos, const float* rsin, const float* alibi,
                               const int* seg, const int* tok, int* status, cudaStream_t st);
// dqkv[:, q heads] = inverse-RoPE(dq_acc / sqrt(Dh)) as bf16 (rcos = null: no rotation);
// rows and positions as launch_rope_apply
cudaError_t launch_dq_finish(const float* dq_acc, bf16* dqkv, int ldqkv, int H, int Dh, const float* rcos,
                             const float* rsin, const int* cnt, int S, int max_rows, const int* tok, cudaStream_t st);

// ------------------------------------------------------------------------
// GEMM: D(m,n) = alpha * sum_k A(m,k) B(n,k) with a fused epilogue.
// ------------------------------------------------------------------------
// EPI_STORE       D = alpha*acc (bf16)        EPI_STORE_F32  D = alpha*acc (float)
// EPI_RESID       x[kept row] += alpha*acc (float32 residual), save = new x (bf16)
// EPI_ROPE        D = rope(acc) on the first rope_cols columns (q and k heads of
//                 the QKV projection, position = row % S), plain store after
// EPI_SWIGLU      B is read as matching halves of the gate and up rows; writes
//                 g, u to D (row stride 2F, columns j and F+j) and
//                 h = silu(g) u to h_out (row stride F)
// EPI_SWIGLU_BWD  acc = dh; with g, u from `gu` writes dg, du to D (stride 2F)
// EPI_RELU2: D = u (bf16 save), h_out = max(u, 0)^2 (both [M, N], row stride ldd);
// EPI_RELU2_BWD: D = dh * 2 max(u, 0) with u read from `gu` ([M, N], stride ldd).
enum EpiMode {
  EPI_STORE = 0,
  EPI_STORE_F32 = 1,
  EPI_RESID = 2,
  EPI_ROPE = 3,
  EPI_SWIGLU = 4,
  EPI_SWIGLU_BWD = 5,
  EPI_RELU2 = 6,
  EPI_RELU2_BWD = 7
};

struct GemmArgs {
  // problem size; a non-null *_cnt makes the extent device-side: (*cnt) * mul
  int M;
  const int* M_cnt;
  int M_mul;
  int N;
  int K;
  const int* K_cnt;
  int K_mul;
  int M_cap, K_cap;  // worst-case extents (tensor maps, grid)
  // operands: A(m,k) = A[m*lda+k] (a_mn=0) or A[k*lda+m] (a_mn=1); same for B(n,k)
  const void* A;
  int lda, a_mn;
  const void* B;
  int ldb, b_mn;
  // epilogue
  int epi;
  void* D;
  int ldd;
  float alpha;
  // EPI_RESID: x[r] = x[r] + alpha*acc for r = src_row(kept_idx, S, m) on the
  // float32 residual stream x; save[m] = new x[r] (float32, compact).
  // Variants: with resid_src the old value is read from the compact copy
  // resid_src[m*ld_src] instead of x[r]; with x_skip the new value goes to
  // save only and x is left as it was.
  float* x;
  int ldx;
  const int* kept_idx;
  int S;
  void* save;
  int ld_save;
  const float* resid_src;
  int ld_src;
  int x_skip;
  // EPI_ROPE (position of row m: row_pos(pos_tok, S, m))
  const float* rope_cos;
  const float* rope_sin;
  int Dh, rope_cols;
  const int* pos_tok;
  // EPI_SWIGLU / EPI_SWIGLU_BWD
  const void* gu;
  void* h_out;
  int F;
  int* status;
};

cudaError_t gemm_tc(const GemmArgs& a, cudaStream_t st);    // bf16 operands, tcgen05
// One block whose bounded wait never completes: records LD_ERR_TIMEOUT.
cudaError_t launch_wait_timeout(int* status, cudaStream_t st);
cudaError_t gemm_simt(const GemmArgs& a, cudaStream_t st);  // float operands, SIMT
int device_sm_count();

}  // namespace ldk
