// Causal grouped-query attention on CUDA cores (float32 arithmetic), the
// attention of the float32 debug path.  One warp per (row, head).
//
// f_attn of Eq. (transformer_layer_dropout_train) for one kept sequence:
//   o_i = sum_{j<=i} softmax_j(c q_i . k_j [+ m_h (j - i)]) v_j,  c = 1/sqrt(Dh),
// (the bracket with an ALiBi slope table), query head h reads key/value head
// floor(h*Hkv/H).  Rows are compact: the
// kept sequence s occupies rows s*S .. s*S+S-1 of qkv, whose columns are
// [Q heads | K heads | V heads].  lse[h][m] = log sum_j exp(c q_m . k_j).
// With per-token kept lists (seg, tok) the kept tokens of sequence b occupy
// rows seg[b] .. seg[b+1]-1 and attend among themselves in that order; rows
// with tok[m] < 0 (padding) belong to no sequence and are skipped.
#include "ld_internal.cuh"

namespace ldk {

// Sequence of compact row m: its first row seq0, its index pos in the
// sequence and the sequence's length; false for a padding row.
__device__ __forceinline__ bool row_seq(long long m, int S, const int* seg, const int* tok, long long& seq0,
                                        int& pos, int& len) {
  if (!seg) {
    seq0 = (m / S) * S;
    pos = (int)(m % S);
    len = S;
    return true;
  }
  const int t = tok[m];
  if (t < 0) return false;
  const int b = t / S;
  seq0 = seg[b];
  pos = (int)(m - seq0);
  len = seg[b + 1] - seg[b];
  return true;
}

__device__ __forceinline__ float wsum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float wmax(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

constexpr int kWarps = 4;

template <typename T>
__global__ void __launch_bounds__(128) attn_fwd_simt_kernel(const T* __restrict__ qkv, int ldq, T* __restrict__ o,
                                                            int ldo, float* __restrict__ lse, int lse_ld,
                                                            const int* __restrict__ cnt, int S, int H, int Hkv,
                                                            int Dh, const float* __restrict__ alibi,
                                                            const int* __restrict__ seg, const int* __restrict__ tok) {
  __shared__ float qs[kWarps][128];
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long M = seg ? (long long)(*cnt) : (long long)(*cnt) * S;
  const float c = 1.0f / sqrtf((float)Dh);
  const int ne = Dh / 32;
  const long long nwarps = (long long)gridDim.x * kWarps;
  for (long long it = (long long)blockIdx.x * kWarps + w; it < M * H; it += nwarps) {
    const long long m = it / H;
    const int h = (int)(it % H);
    long long seq0;
    int pos, len;
    if (!row_seq(m, S, seg, tok, seq0, pos, len)) continue;
    const int g = (h * Hkv) / H;
    for (int i = lane; i < Dh; i += 32) qs[w][i] = c * to_f(qkv[m * ldq + (long long)h * Dh + i]);
    __syncwarp();
    float mx = -INFINITY, sum = 0.f, acc[4] = {0.f, 0.f, 0.f, 0.f};
    for (int j0 = 0; j0 <= pos; j0 += 32) {
      const int j = j0 + lane;
      float s = -INFINITY;
      if (j <= pos) {
        const T* kr = qkv + (seq0 + j) * ldq + (long long)(H + g) * Dh;
        float t = 0.f;
        for (int i = 0; i < Dh; ++i) t += qs[w][i] * to_f(kr[i]);
        s = alibi ? t + alibi[h] * (float)(j - pos) : t;
      }
      const float nmx = fmaxf(mx, wmax(s));
      const float p = (j <= pos) ? expf(s - nmx) : 0.f;
      const float corr = expf(mx - nmx);
      sum = sum * corr + wsum(p);
      for (int e = 0; e < ne; ++e) acc[e] *= corr;
      const int jend = min(32, pos - j0 + 1);
      for (int jj = 0; jj < jend; ++jj) {
        const float pj = __shfl_sync(0xffffffffu, p, jj);
        const T* vr = qkv + (seq0 + j0 + jj) * ldq + (long long)(H + Hkv + g) * Dh;
        for (int e = 0; e < ne; ++e) acc[e] += pj * to_f(vr[lane + 32 * e]);
      }
      mx = nmx;
    }
    for (int e = 0; e < ne; ++e) o[m * ldo + (long long)h * Dh + lane + 32 * e] = from_f<T>(acc[e] / sum);
    if (lane == 0) lse[(size_t)h * lse_ld + m] = mx + logf(sum);
    __syncwarp();
  }
}

// dq_i = c sum_{j<=i} dS_ij k_j with dS_ij = P_ij (dO_i . v_j - D_i).
template <typename T>
__global__ void __launch_bounds__(128) attn_dq_simt_kernel(const T* __restrict__ qkv, int ldq,
                                                           const T* __restrict__ dO, int ldo,
                                                           const float* __restrict__ lse,
                                                           const float* __restrict__ Dvec, int lse_ld,
                                                           T* __restrict__ dqkv, const int* __restrict__ cnt, int S,
                                                           int H, int Hkv, int Dh, const float* __restrict__ alibi,
                                                           const int* __restrict__ seg, const int* __restrict__ tok) {
  __shared__ float qs[kWarps][128];
  __shared__ float ds_[kWarps][128];
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long M = seg ? (long long)(*cnt) : (long long)(*cnt) * S;
  const float c = 1.0f / sqrtf((float)Dh);
  const int ne = Dh / 32;
  const long long nwarps = (long long)gridDim.x * kWarps;
  for (long long it = (long long)blockIdx.x * kWarps + w; it < M * H; it += nwarps) {
    const long long m = it / H;
    const int h = (int)(it % H);
    long long seq0;
    int pos, len;
    if (!row_seq(m, S, seg, tok, seq0, pos, len)) continue;
    const int g = (h * Hkv) / H;
    for (int i = lane; i < Dh; i += 32) {
      qs[w][i] = c * to_f(qkv[m * ldq + (long long)h * Dh + i]);
      ds_[w][i] = to_f(dO[m * ldo + (long long)h * Dh + i]);
    }
    __syncwarp();
    const float L_ = lse[(size_t)h * lse_ld + m], D_ = Dvec[(size_t)h * lse_ld + m];
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
    for (int j0 = 0; j0 <= pos; j0 += 32) {
      const int j = j0 + lane;
      float dsv = 0.f;
      if (j <= pos) {
        const T* kr = qkv + (seq0 + j) * ldq + (long long)(H + g) * Dh;
        const T* vr = qkv + (seq0 + j) * ldq + (long long)(H + Hkv + g) * Dh;
        float s = 0.f, dp = 0.f;
        for (int i = 0; i < Dh; ++i) {
          s += qs[w][i] * to_f(kr[i]);
          dp += ds_[w][i] * to_f(vr[i]);
        }
        if (alibi) s += alibi[h] * (float)(j - pos);
        const float p = expf(s - L_);
        dsv = p * (dp - D_);
      }
      const int jend = min(32, pos - j0 + 1);
      for (int jj = 0; jj < jend; ++jj) {
        const float dj = __shfl_sync(0xffffffffu, dsv, jj);
        const T* kr = qkv + (seq0 + j0 + jj) * ldq + (long long)(H + g) * Dh;
        for (int e = 0; e < ne; ++e) acc[e] += dj * to_f(kr[lane + 32 * e]);
      }
    }
    for (int e = 0; e < ne; ++e) dqkv[m * ldq + (long long)h * Dh + lane + 32 * e] = from_f<T>(c * acc[e]);
    __syncwarp();
  }
}

// dk_j = c sum_{h in group} sum_{i>=j} dS_ij q_i ;  dv_j = sum_h sum_{i>=j} P_ij dO_i.
template <typename T>
__global__ void __launch_bounds__(128) attn_dkv_simt_kernel(const T* __restrict__ qkv, int ldq,
                                                            const T* __restrict__ dO, int ldo,
                                                            const float* __restrict__ lse,
                                                            const float* __restrict__ Dvec, int lse_ld,
                                                            T* __restrict__ dqkv, const int* __restrict__ cnt,
                                                            int S, int H, int Hkv, int Dh,
                                                            const float* __restrict__ alibi,
                                                            const int* __restrict__ seg, const int* __restrict__ tok) {
  __shared__ float ks[kWarps][128];
  __shared__ float vs[kWarps][128];
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long M = seg ? (long long)(*cnt) : (long long)(*cnt) * S;
  const float c = 1.0f / sqrtf((float)Dh);
  const int ne = Dh / 32;
  const int grp = H / Hkv;
  const long long nwarps = (long long)gridDim.x * kWarps;
  for (long long it = (long long)blockIdx.x * kWarps + w; it < M * Hkv; it += nwarps) {
    const long long mk = it / Hkv;
    const int g = (int)(it % Hkv);
    long long seq0;
    int pos, len;
    if (!row_seq(mk, S, seg, tok, seq0, pos, len)) continue;
    for (int i = lane; i < Dh; i += 32) {
      ks[w][i] = c * to_f(qkv[mk * ldq + (long long)(H + g) * Dh + i]);
      vs[w][i] = to_f(qkv[mk * ldq + (long long)(H + Hkv + g) * Dh + i]);
    }
    __syncwarp();
    float dk[4] = {0.f, 0.f, 0.f, 0.f}, dv[4] = {0.f, 0.f, 0.f, 0.f};
    for (int h = g * grp; h < (g + 1) * grp; ++h) {
      for (int i0 = pos; i0 < len; i0 += 32) {
        const int i = i0 + lane;
        float p = 0.f, dsv = 0.f;
        if (i < len) {
          const long long mq = seq0 + i;
          const T* qr = qkv + mq * ldq + (long long)h * Dh;
          const T* dr = dO + mq * ldo + (long long)h * Dh;
          float s = 0.f, dp = 0.f;
          for (int e = 0; e < Dh; ++e) {
            s += ks[w][e] * to_f(qr[e]);
            dp += vs[w][e] * to_f(dr[e]);
          }
          if (alibi) s += alibi[h] * (float)(pos - i);
          p = expf(s - lse[(size_t)h * lse_ld + mq]);
          dsv = p * (dp - Dvec[(size_t)h * lse_ld + mq]);
        }
        const int iend = min(32, len - i0);
        for (int ii = 0; ii < iend; ++ii) {
          const float pi = __shfl_sync(0xffffffffu, p, ii);
          const float di = __shfl_sync(0xffffffffu, dsv, ii);
          const long long mq = seq0 + i0 + ii;
          const T* qr = qkv + mq * ldq + (long long)h * Dh;
          const T* dr = dO + mq * ldo + (long long)h * Dh;
          for (int e = 0; e < ne; ++e) {
            dk[e] += di * to_f(qr[lane + 32 * e]);
            dv[e] += pi * to_f(dr[lane + 32 * e]);
          }
        }
      }
    }
    for (int e = 0; e < ne; ++e) {
      dqkv[mk * ldq + (long long)(H + g) * Dh + lane + 32 * e] = from_f<T>(c * dk[e]);
      dqkv[mk * ldq + (long long)(H + Hkv + g) * Dh + lane + 32 * e] = from_f<T>(dv[e]);
    }
    __syncwarp();
  }
}

static int attn_grid(long long items) {
  long long g = (items + kWarps - 1) / kWarps;
  const long long cap = (long long)device_sm_count() * 32;
  if (g > cap) g = cap;
  if (g < 1) g = 1;
  return (int)g;
}

template <typename T>
cudaError_t launch_attn_fwd_simt(const T* qkv, int ldqkv, T* o, int ldo, float* lse, const int* cnt, int S, int H,
                                 int Hkv, int Dh, int max_rows, const float* alibi, const int* seg, const int* tok,
                                 cudaStream_t st) {
  attn_fwd_simt_kernel<T><<<attn_grid((long long)max_rows * H), 128, 0, st>>>(qkv, ldqkv, o, ldo, lse, max_rows,
                                                                               cnt, S, H, Hkv, Dh, alibi, seg, tok);
  return cudaGetLastError();
}

template <typename T>
cudaError_t launch_attn_bwd_simt(const T* qkv, int ldqkv, const T* dO, int ldo, const float* lse, const float* Dvec,
                                 T* dqkv, const int* cnt, int S, int H, int Hkv, int Dh, int max_rows,
                                 const float* alibi, const int* seg, const int* tok, cudaStream_t st) {
  attn_dq_simt_kernel<T><<<attn_grid((long long)max_rows * H), 128, 0, st>>>(
      qkv, ldqkv, dO, ldo, lse, Dvec, max_rows, dqkv, cnt, S, H, Hkv, Dh, alibi, seg, tok);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  attn_dkv_simt_kernel<T><<<attn_grid((long long)max_rows * Hkv), 128, 0, st>>>(
      qkv, ldqkv, dO, ldo, lse, Dvec, max_rows, dqkv, cnt, S, H, Hkv, Dh, alibi, seg, tok);
  return cudaGetLastError();
}

template cudaError_t launch_attn_fwd_simt<float>(const float*, int, float*, int, float*, const int*, int, int, int,
                                                 int, int, const float*, const int*, const int*, cudaStream_t);
template cudaError_t launch_attn_fwd_simt<bf16>(const bf16*, int, bf16*, int, float*, const int*, int, int, int, int,
                                                int, const float*, const int*, const int*, cudaStream_t);
template cudaError_t launch_attn_bwd_simt<float>(const float*, int, const float*, int, const float*, const float*,
                                                 float*, const int*, int, int, int, int, int, const float*,
                                                 const int*, const int*, cudaStream_t);
template cudaError_t launch_attn_bwd_simt<bf16>(const bf16*, int, const bf16*, int, const float*, const float*, bf16*,
                                                const int*, int, int, int, int, int, const float*, const int*,
                                                const int*, cudaStream_t);

}  // namespace ldk
