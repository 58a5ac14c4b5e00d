// float32 GEMM on CUDA cores for the debug path:
//   D(m,n) = alpha * sum_k A(m,k) B(n,k)
// with the same epilogues as the tensor-core GEMM (plain store, or the
// scaled residual update written back to the kept rows of the residual
// stream).  64x64 tiles, 256 threads, 4x4 outputs per thread.
#include "ld_internal.cuh"

namespace ldk {

template <int EPI>
__global__ void __launch_bounds__(256) gemm_simt_kernel(const GemmArgs a) {
  const int M = a.M_cnt ? (*a.M_cnt) * a.M_mul : a.M;
  const int K = a.K_cnt ? (*a.K_cnt) * a.K_mul : a.K;
  const int N = a.N;
  const int m0 = blockIdx.x * 64, n0 = blockIdx.y * 64;
  if (m0 >= M || n0 >= N) return;
  __shared__ float As[16][68];
  __shared__ float Bs[16][68];
  const float* A = static_cast<const float*>(a.A);
  const float* B = static_cast<const float*>(a.B);
  const int tid = threadIdx.x, ty = tid / 16, tx = tid % 16;
  float acc[4][4] = {};
  for (int k0 = 0; k0 < K; k0 += 16) {
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int e = tid * 4 + r;
      int mm, kk;
      if (a.a_mn) { kk = e / 64; mm = e % 64; } else { mm = e / 16; kk = e % 16; }
      const int m = m0 + mm, k = k0 + kk;
      float v = 0.f;
      if (m < M && k < K) v = a.a_mn ? A[(size_t)k * a.lda + m] : A[(size_t)m * a.lda + k];
      As[kk][mm] = v;
      int nn, kb;
      if (a.b_mn) { kb = e / 64; nn = e % 64; } else { nn = e / 16; kb = e % 16; }
      const int n = n0 + nn, kx = k0 + kb;
      float w = 0.f;
      if (n < N && kx < K) w = a.b_mn ? B[(size_t)kx * a.ldb + n] : B[(size_t)n * a.ldb + kx];
      Bs[kb][nn] = w;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < 16; ++kk) {
      float av[4], bv[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        av[i] = As[kk][ty * 4 + i];
        bv[i] = Bs[kk][tx * 4 + i];
      }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] += av[i] * bv[j];
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int m = m0 + ty * 4 + i;
    if (m >= M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = n0 + tx * 4 + j;
      if (n >= N) continue;
      const float v = a.alpha * acc[i][j];
      if (EPI == EPI_RESID) {
        const long long r = src_row(a.kept_idx, a.S, m);
        if (r < 0) {  // padding row of a per-token kept list: zero copy only
          if (a.save) static_cast<float*>(a.save)[(size_t)m * a.ld_save + n] = 0.f;
          continue;
        }
        float* x = a.x + r * a.ldx + n;
        const float nv = (a.resid_src ? a.resid_src[(size_t)m * a.ld_src + n] : *x) + v;
        if (!a.x_skip) *x = nv;
        if (a.save) static_cast<float*>(a.save)[(size_t)m * a.ld_save + n] = nv;
      } else {
        static_cast<float*>(a.D)[(size_t)m * a.ldd + n] = v;
      }
    }
  }
}

cudaError_t gemm_simt(const GemmArgs& a, cudaStream_t st) {
  const int mcap = a.M_cnt ? a.M_cap : a.M;
  dim3 grid((mcap + 63) / 64, (a.N + 63) / 64);
  if (grid.x == 0 || grid.y == 0) return cudaSuccess;
  if (a.epi == EPI_RESID)
    gemm_simt_kernel<EPI_RESID><<<grid, 256, 0, st>>>(a);
  else
    gemm_simt_kernel<EPI_STORE_F32><<<grid, 256, 0, st>>>(a);
  return cudaGetLastError();
}

}  // namespace ldk
