// Row-wise kernels of the layer (HBM-bound): RMSNorm forward with the
// kept-row gather, RMSNorm backward with the in-place residual gradient,
// the scaled gather of the upstream gradient, RoPE, SwiGLU and small
// reductions.  All of them read the kept count of their layer from device
// memory and walk compact rows m < kept_cnt * S with a grid-stride loop, so
// no launch depends on a host-side copy of the masks.
#include "ld_internal.cuh"

namespace ldk {

// 8 consecutive elements <-> 8 floats (16 bytes of bf16, 32 bytes of float).
__device__ __forceinline__ void ld8(const bf16* p, float* v) {
  const uint4 r = *reinterpret_cast<const uint4*>(p);
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&r);
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const float2 f = __bfloat1622float2(h[j]);
    v[2 * j] = f.x;
    v[2 * j + 1] = f.y;
  }
}
__device__ __forceinline__ void ld8(const float* p, float* v) {
  const float4 a = reinterpret_cast<const float4*>(p)[0];
  const float4 b = reinterpret_cast<const float4*>(p)[1];
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
  v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}
__device__ __forceinline__ void st8(bf16* p, const float* v) {
  uint4 r;
  __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&r);
#pragma unroll
  for (int j = 0; j < 4; ++j) h[j] = __floats2bfloat162_rn(v[2 * j], v[2 * j + 1]);
  *reinterpret_cast<uint4*>(p) = r;
}
__device__ __forceinline__ void st8(float* p, const float* v) {
  reinterpret_cast<float4*>(p)[0] = make_float4(v[0], v[1], v[2], v[3]);
  reinterpret_cast<float4*>(p)[1] = make_float4(v[4], v[5], v[6], v[7]);
}
// Round to the storage type and back (the value that st8 would store).
__device__ __forceinline__ float rnd(float v, const bf16*) { return __bfloat162float(__float2bfloat16_rn(v)); }
__device__ __forceinline__ float rnd(float v, const float*) { return v; }

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

static int grid_for(long long work_items, int per_block, int cap) {
  long long g = (work_items + per_block - 1) / per_block;
  if (g < 1) g = 1;
  if (g > cap) g = cap;
  return (int)g;
}
int device_sm_count() {
  // once per process (initialisation of a function-local static is thread-safe)
  static const int n = [] {
    int dev = 0, v = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev);
    return v > 0 ? v : 152;
  }();
  return n;
}

// ---------------------------------------------------------------- RMSNorm fwd
template <typename TS, typename T>
__global__ void __launch_bounds__(256) rmsnorm_fwd_kernel(const TS* __restrict__ src, int gather,
                                                          const int* __restrict__ kept_idx,
                                                          const int* __restrict__ cnt, int S, int d,
                                                          const T* __restrict__ gamma, float eps,
                                                          TS* __restrict__ copy, T* __restrict__ out,
                                                          float* __restrict__ rstd) {
  const long long M = (long long)(*cnt) * S;
  const int lane = threadIdx.x & 31;
  const long long nwarps = (long long)gridDim.x * (blockDim.x >> 5);
  for (long long m = (long long)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); m < M; m += nwarps) {
    const long long r = gather ? src_row(kept_idx, S, m) : m;
    if (r < 0) {  // padding row of a per-token kept list: zeros
      const float z[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
      for (int i = lane * 8; i < d; i += 256) {
        if (copy) st8(copy + m * d + i, z);
        st8(out + m * d + i, z);
      }
      if (lane == 0) rstd[m] = 0.f;
      continue;
    }
    const TS* xr = src + r * d;
    float ss = 0.f;
    for (int i = lane * 8; i < d; i += 256) {
      float v[8];
      ld8(xr + i, v);
#pragma unroll
      for (int j = 0; j < 8; ++j) ss += v[j] * v[j];
      if (copy) st8(copy + m * d + i, v);
    }
    ss = warp_sum(ss);
    const float rs = 1.0f / sqrtf(ss / (float)d + eps);
    if (lane == 0) rstd[m] = rs;
    for (int i = lane * 8; i < d; i += 256) {
      float v[8], g[8], o[8];
      ld8(xr + i, v);
      ld8(gamma + i, g);
#pragma unroll
      for (int j = 0; j < 8; ++j) o[j] = (v[j] * rs) * g[j];
      st8(out + m * d + i, o);
    }
  }
}

// As rmsnorm_fwd_kernel for d <= 256 NV, with each warp's row held in
// registers (NV vectors of 8 per lane), so the row is read from memory once:
// the two-pass form re-reads it after the sum of squares, and with tens of
// thousands of rows in flight the second read misses L2 (measured at the
// Llama-3-8B width: DRAM reads twice the row bytes).  Four warps a block and
// few blocks per SM still keep ~16 KB a warp in flight.
template <typename TS, typename T, int NV>
__global__ void __launch_bounds__(128) rmsnorm_fwd_reg_kernel(const TS* __restrict__ src, int gather,
                                                              const int* __restrict__ kept_idx,
                                                              const int* __restrict__ cnt, int S, int d,
                                                              const T* __restrict__ gamma, float eps,
                                                              TS* __restrict__ copy, T* __restrict__ out,
                                                              float* __restrict__ rstd) {
  const long long M = (long long)(*cnt) * S;
  const int lane = threadIdx.x & 31;
  const long long nwarps = (long long)gridDim.x * (blockDim.x >> 5);
  for (long long m = (long long)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); m < M; m += nwarps) {
    const long long r = gather ? src_row(kept_idx, S, m) : m;
    if (r < 0) {  // padding row of a per-token kept list: zeros
      const float z[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
      for (int i = lane * 8; i < d; i += 256) {
        if (copy) st8(copy + m * d + i, z);
        st8(out + m * d + i, z);
      }
      if (lane == 0) rstd[m] = 0.f;
      continue;
    }
    const TS* xr = src + r * d;
    float v[NV][8];
#pragma unroll
    for (int j = 0; j < NV; ++j)
      if (lane * 8 + 256 * j < d) ld8(xr + lane * 8 + 256 * j, v[j]);
    float ss = 0.f;
#pragma unroll
    for (int j = 0; j < NV; ++j)
      if (lane * 8 + 256 * j < d) {
#pragma unroll
        for (int e = 0; e < 8; ++e) ss += v[j][e] * v[j][e];
        if (copy) st8(copy + m * d + lane * 8 + 256 * j, v[j]);
      }
    ss = warp_sum(ss);
    const float rs = 1.0f / sqrtf(ss / (float)d + eps);
    if (lane == 0) rstd[m] = rs;
#pragma unroll
    for (int j = 0; j < NV; ++j)
      if (lane * 8 + 256 * j < d) {
        float g[8], o[8];
        ld8(gamma + lane * 8 + 256 * j, g);
#pragma unroll
        for (int e = 0; e < 8; ++e) o[e] = (v[j][e] * rs) * g[e];
        st8(out + m * d + lane * 8 + 256 * j, o);
      }
  }
}

template <typename TS, typename T>
cudaError_t launch_rmsnorm_fwd(const TS* src, int gather, const int* kept_idx, const int* cnt, int S, int d,
                               int max_rows, const T* gamma, float eps, TS* copy, T* out, float* rstd,
                               cudaStream_t st) {
  if (d <= 4096) {
    // 4 rows a block, up to 8 blocks per SM
    const int grid = grid_for(max_rows, 4, device_sm_count() * 8);
    if (d <= 1024)
      rmsnorm_fwd_reg_kernel<TS, T, 4><<<grid, 128, 0, st>>>(src, gather, kept_idx, cnt, S, d, gamma, eps, copy, out,
                                                              rstd);
    else if (d <= 2048)
      rmsnorm_fwd_reg_kernel<TS, T, 8><<<grid, 128, 0, st>>>(src, gather, kept_idx, cnt, S, d, gamma, eps, copy, out,
                                                              rstd);
    else
      rmsnorm_fwd_reg_kernel<TS, T, 16><<<grid, 128, 0, st>>>(src, gather, kept_idx, cnt, S, d, gamma, eps, copy,
                                                               out, rstd);
    return cudaGetLastError();
  }
  const int grid = grid_for(max_rows, 8, device_sm_count() * 16);
  rmsnorm_fwd_kernel<TS, T><<<grid, 256, 0, st>>>(src, gather, kept_idx, cnt, S, d, gamma, eps, copy, out, rstd);
  return cudaGetLastError();
}

// ---------------------------------------------------------------- RMSNorm bwd
template <typename T>
__global__ void __launch_bounds__(256) rmsnorm_bwd_kernel(const float* __restrict__ dyn, const float* __restrict__ xs,
                                                          const float* __restrict__ rstd,
                                                          const T* __restrict__ gamma, float* __restrict__ dx,
                                                          const int* __restrict__ kept_idx,
                                                          const int* __restrict__ cnt, int S, int d, float scale,
                                                          T* __restrict__ next, float* __restrict__ part) {
  extern __shared__ float sg[];  // partial gain gradient of this block, [d]
  for (int i = threadIdx.x; i < d; i += blockDim.x) sg[i] = 0.f;
  __syncthreads();
  const long long M = (long long)(*cnt) * S;
  const int lane = threadIdx.x & 31;
  const long long nwarps = (long long)gridDim.x * (blockDim.x >> 5);
  for (long long m = (long long)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); m < M; m += nwarps) {
    const long long r = src_row(kept_idx, S, m);
    const float rs = rstd[m];
    float dot = 0.f;
    for (int i = lane * 8; i < d; i += 256) {
      float dy[8], xv[8], g[8];
      ld8(dyn + m * d + i, dy);
      ld8(xs + m * d + i, xv);
      ld8(gamma + i, g);
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const float xn = xv[j] * rs;
        dot += dy[j] * g[j] * xn;
        atomicAdd(&sg[i + j], dy[j] * xn);
      }
    }
    dot = warp_sum(dot) / (float)d;
    if (r < 0) {  // padding row of a per-token kept list (its dyn and xs are 0)
      const float z[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
      if (next)
        for (int i = lane * 8; i < d; i += 256) st8(next + m * d + i, z);
      continue;
    }
    for (int i = lane * 8; i < d; i += 256) {
      float dy[8], xv[8], g[8], cur[8], nx[8];
      ld8(dyn + m * d + i, dy);
      ld8(xs + m * d + i, xv);
      ld8(gamma + i, g);
      ld8(dx + r * d + i, cur);
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const float xn = xv[j] * rs;
        cur[j] = cur[j] + rs * (dy[j] * g[j] - xn * dot);
        nx[j] = scale * cur[j];
      }
      st8(dx + r * d + i, cur);
      if (next) st8(next + m * d + i, nx);
    }
  }
  __syncthreads();
  for (int i = threadIdx.x; i < d; i += blockDim.x) part[(size_t)blockIdx.x * d + i] = sg[i];
}

int rmsnorm_bwd_blocks(int max_rows) { return grid_for(max_rows, 8, device_sm_count() * 2); }

// Same operation with the block spread over the columns: thread t owns the
// 8-column chunks t, t + 256, ... (MAXJ of them), keeps its share of gamma and
// of the gain gradient in registers, and the block reduces the dot products of
// RPB rows at once (their loads are all in flight together).  No
// shared-memory atomics; all global accesses coalesced.
// PF: the residual-gradient rows dx are read together with dyn and xs (one
// memory round trip per row group instead of two; costs 8 MAXJ RPB registers).
template <typename T, int MAXJ, int RPB, bool PF>
__global__ void __launch_bounds__(256) rmsnorm_bwd_cols_kernel(const float* __restrict__ dyn,
                                                               const float* __restrict__ xs,
                                                               const float* __restrict__ rstd,
                                                               const T* __restrict__ gamma, float* __restrict__ dx,
                                                               const int* __restrict__ kept_idx,
                                                               const int* __restrict__ cnt, int S, int d, float scale,
                                                               T* __restrict__ next, float* __restrict__ part) {
  __shared__ float red[RPB][8];
  __shared__ float tot[RPB];
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  const int d8 = d / 8;
  float g[MAXJ][8], gacc[MAXJ][8];
#pragma unroll
  for (int j = 0; j < MAXJ; ++j) {
    const int c8 = tid + 256 * j;
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      g[j][e] = 0.f;
      gacc[j][e] = 0.f;
    }
    if (c8 < d8) ld8(gamma + c8 * 8, g[j]);
  }
  const long long M = (long long)(*cnt) * S;
  for (long long m0 = (long long)blockIdx.x * RPB; m0 < M; m0 += (long long)gridDim.x * RPB) {
    float dy[RPB][MAXJ][8], xv[RPB][MAXJ][8], cur[PF ? RPB : 1][MAXJ][8];
    float pd[RPB];
    long long rr[RPB];
#pragma unroll
    for (int q = 0; q < RPB; ++q) rr[q] = (m0 + q < M) ? src_row(kept_idx, S, m0 + q) : -1;
#pragma unroll
    for (int q = 0; q < RPB; ++q) {
      const long long m = m0 + q;
      pd[q] = 0.f;
#pragma unroll
      for (int j = 0; j < MAXJ; ++j) {
        const int c8 = tid + 256 * j;
        if (m < M && c8 < d8) {
          ld8(dyn + m * d + c8 * 8, dy[q][j]);
          ld8(xs + m * d + c8 * 8, xv[q][j]);
          if constexpr (PF) {
            if (rr[q] >= 0) {
              ld8(dx + rr[q] * d + c8 * 8, cur[q][j]);
            } else {
#pragma unroll
              for (int e = 0; e < 8; ++e) cur[q][j][e] = 0.f;
            }
          }
#pragma unroll
          for (int e = 0; e < 8; ++e) pd[q] += dy[q][j][e] * g[j][e] * xv[q][j][e];
        }
      }
    }
#pragma unroll
    for (int q = 0; q < RPB; ++q) {
      const float v = warp_sum(pd[q]);
      if (lane == 0) red[q][w] = v;
    }
    __syncthreads();
    if (w < RPB) {
      float v = lane < 8 ? red[w][lane] : 0.f;
      v = warp_sum(v);
      if (lane == 0) tot[w] = v;
    }
    __syncthreads();
#pragma unroll
    for (int q = 0; q < RPB; ++q) {
      const long long m = m0 + q;
      if (m >= M) break;
      const long long r = rr[q];
      const float rs = rstd[m];
      const float dot = tot[q] * rs / (float)d;  // mean(dyn * gamma * xn)
#pragma unroll
      for (int j = 0; j < MAXJ; ++j) {
        const int c8 = tid + 256 * j;
        if (c8 < d8) {
          float cr[8], nx[8];
          if constexpr (PF) {
#pragma unroll
            for (int e = 0; e < 8; ++e) cr[e] = cur[q][j][e];
          } else if (r >= 0) {
            ld8(dx + r * d + c8 * 8, cr);
          } else {
#pragma unroll
            for (int e = 0; e < 8; ++e) cr[e] = 0.f;
          }
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const float xn = xv[q][j][e] * rs;
            cr[e] = cr[e] + rs * (dy[q][j][e] * g[j][e] - xn * dot);
            nx[e] = scale * cr[e];
            gacc[j][e] += dy[q][j][e] * xn;
          }
          // a padding row of a per-token kept list (r < 0) has dyn = xs = 0:
          // it adds nothing to the gain gradient and passes 0 on
          if (r >= 0) st8(dx + r * d + c8 * 8, cr);
          if (next) st8(next + m * d + c8 * 8, nx);
        }
      }
    }
    __syncthreads();  // red / tot are rewritten by the next group
  }
#pragma unroll
  for (int j = 0; j < MAXJ; ++j) {
    const int c8 = tid + 256 * j;
    if (c8 < d8) st8(part + (size_t)blockIdx.x * d + c8 * 8, gacc[j]);
  }
}

template <typename T>
cudaError_t launch_rmsnorm_bwd(const float* dyn, const float* xs, const float* rstd, const T* gamma, float* dx,
                               const int* kept_idx, const int* cnt, int S, int d, int max_rows, float scale,
                               T* next, float* part, int nblocks, cudaStream_t st) {
  (void)max_rows;
  if (d <= 2048) {
    rmsnorm_bwd_cols_kernel<T, 1, 2, true><<<nblocks, 256, 0, st>>>(dyn, xs, rstd, gamma, dx, kept_idx, cnt, S, d, scale, next, part);
  } else if (d <= 4096) {
    rmsnorm_bwd_cols_kernel<T, 2, 1, true><<<nblocks, 256, 0, st>>>(dyn, xs, rstd, gamma, dx, kept_idx, cnt, S, d, scale, next, part);
  } else if (d <= 8192) {
    rmsnorm_bwd_cols_kernel<T, 4, 1, false><<<nblocks, 256, 0, st>>>(dyn, xs, rstd, gamma, dx, kept_idx, cnt, S, d, scale, next, part);
  } else {
    const size_t smem = (size_t)d * sizeof(float);
    if (smem > 48 * 1024) {
      cudaError_t e = cudaFuncSetAttribute(rmsnorm_bwd_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)smem);
      if (e != cudaSuccess) return e;
    }
    rmsnorm_bwd_kernel<T><<<nblocks, 256, smem, st>>>(dyn, xs, rstd, gamma, dx, kept_idx, cnt, S, d, scale, next,
                                                     part);
  }
  return cudaGetLastError();
}

// out[c] = sum over rows of part[row][c]: a block owns 32 columns, its 8
// warps take every 8th row (one coalesced 128-byte read per warp and row),
// and the 8 partial sums are combined in shared memory.
__global__ void __launch_bounds__(256) colsum_kernel(const float* __restrict__ part, int nrows, int d,
                                                     float* __restrict__ out) {
  __shared__ float red[8][33];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int c = blockIdx.x * 32 + lane;
  float s = 0.f;
  if (c < d)
    for (int r = w; r < nrows; r += 8) s += part[(size_t)r * d + c];
  red[w][lane] = s;
  __syncthreads();
  if (w == 0 && c < d) {
    float t = 0.f;
#pragma unroll
    for (int k = 0; k < 8; ++k) t += red[k][lane];
    out[c] = t;
  }
}

cudaError_t launch_colsum(const float* part, int nrows, int d, float* out, cudaStream_t st) {
  colsum_kernel<<<(d + 31) / 32, 256, 0, st>>>(part, nrows, d, out);
  return cudaGetLastError();
}

// ------------------------------------------------------------- scaled gather
template <typename T>
__global__ void gather_scale_kernel(const float* __restrict__ dx, const int* __restrict__ kept_idx,
                                    const int* __restrict__ cnt, int S, int d, float scale, T* __restrict__ out) {
  const long long M = (long long)(*cnt) * S;
  const int per_row = d / 8;
  const long long total = M * per_row;
  for (long long w = (long long)blockIdx.x * blockDim.x + threadIdx.x; w < total;
       w += (long long)gridDim.x * blockDim.x) {
    const long long m = w / per_row;
    const int i = (int)(w % per_row) * 8;
    float v[8];
    const long long r = src_row(kept_idx, S, m);
    if (r >= 0) {
      ld8(dx + r * d + i, v);
#pragma unroll
      for (int j = 0; j < 8; ++j) v[j] *= scale;
    } else {  // padding row of a per-token kept list
#pragma unroll
      for (int j = 0; j < 8; ++j) v[j] = 0.f;
    }
    st8(out + m * d + i, v);
  }
}

template <typename T>
cudaError_t launch_gather_scale(const float* dx, const int* kept_idx, const int* cnt, int S, int d, int max_rows,
                                float scale, T* out, cudaStream_t st) {
  const int grid = grid_for((long long)max_rows * (d / 8), 256, device_sm_count() * 8);
  gather_scale_kernel<T><<<grid, 256, 0, st>>>(dx, kept_idx, cnt, S, d, scale, out);
  return cudaGetLastError();
}

// ---------------------------------------------------------------- conversion
template <typename TI, typename TO>
__global__ void convert_kernel(const TI* __restrict__ src, TO* __restrict__ dst, long long n8) {
  for (long long w = (long long)blockIdx.x * blockDim.x + threadIdx.x; w < n8; w += (long long)gridDim.x * blockDim.x) {
    float v[8];
    ld8(src + w * 8, v);
    st8(dst + w * 8, v);
  }
}

cudaError_t launch_convert(const void* src, int src_f32, void* dst, int dst_f32, long long n, cudaStream_t st) {
  const long long n8 = n / 8;
  const int grid = grid_for(n8, 256, device_sm_count() * 8);
  if (src_f32 && !dst_f32)
    convert_kernel<float, bf16><<<grid, 256, 0, st>>>(static_cast<const float*>(src), static_cast<bf16*>(dst), n8);
  else if (!src_f32 && dst_f32)
    convert_kernel<bf16, float><<<grid, 256, 0, st>>>(static_cast<const bf16*>(src), static_cast<float*>(dst), n8);
  else
    return cudaMemcpyAsync(dst, src, n * (src_f32 ? 4 : 2), cudaMemcpyDeviceToDevice, st);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------- RoPE
// cos/sin of pos * theta^(-2i/Dh), angles formed in double precision.
__global__ void rope_table_kernel(float* cos_t, float* sin_t, int S, int Dh, double theta) {
  const int half = Dh / 2;
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= S * half) return;
  const int pos = idx / half, i = idx % half;
  const double ang = (double)pos * pow(theta, -(2.0 * i) / (double)Dh);
  double s, c;
  sincos(ang, &s, &c);
  cos_t[idx] = (float)c;
  sin_t[idx] = (float)s;
}

cudaError_t launch_rope_table(float* cos_t, float* sin_t, int S, int Dh, double theta, cudaStream_t st) {
  const int n = S * (Dh / 2);
  rope_table_kernel<<<(n + 255) / 256, 256, 0, st>>>(cos_t, sin_t, S, Dh, theta);
  return cudaGetLastError();
}

// Rotate pairs (i, i+Dh/2) of the first `nheads` heads of each row, at the
// row's position in its sequence; inverse = 1 applies the transpose.  One
// thread per 8 consecutive pairs (16-byte accesses).
template <typename T>
__global__ void rope_apply_kernel(T* __restrict__ qkv, int ld, int nheads, int Dh, const float* __restrict__ cos_t,
                                  const float* __restrict__ sin_t, const int* __restrict__ cnt, int S,
                                  int inverse, const int* __restrict__ tok) {
  const long long M = tok ? (long long)(*cnt) : (long long)(*cnt) * S;
  const int half = Dh / 2, g8 = half / 8;
  const int per_row = nheads * g8;
  const long long total = M * per_row;
  for (long long w = (long long)blockIdx.x * blockDim.x + threadIdx.x; w < total;
       w += (long long)gridDim.x * blockDim.x) {
    const long long m = w / per_row;
    const int rem = (int)(w - m * per_row);
    const int h = rem / g8, i = (rem - h * g8) * 8;
    const int pos = row_pos(tok, S, m);
    T* p = qkv + m * ld + (long long)h * Dh;
    float a[8], b[8], c[8], sn[8];
    ld8(p + i, a);
    ld8(p + half + i, b);
    ld8(cos_t + pos * half + i, c);
    ld8(sin_t + pos * half + i, sn);
    float na[8], nb[8];
    const float sg = inverse ? -1.f : 1.f;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const float s = sg * sn[j];
      na[j] = a[j] * c[j] - b[j] * s;
      nb[j] = b[j] * c[j] + a[j] * s;
    }
    st8(p + i, na);
    st8(p + half + i, nb);
  }
}

template <typename T>
cudaError_t launch_rope_apply(T* qkv, int ld, int nheads, int Dh, const float* cos_t, const float* sin_t,
                              const int* cnt, int S, int max_rows, int inverse, const int* tok, cudaStream_t st) {
  const int grid = grid_for((long long)max_rows * nheads * (Dh / 16), 256, device_sm_count() * 8);
  rope_apply_kernel<T><<<grid, 256, 0, st>>>(qkv, ld, nheads, Dh, cos_t, sin_t, cnt, S, inverse, tok);
  return cudaGetLastError();
}

// ------------------------------------------------------------- zero rows
template <typename T>
__global__ void zero_rows_kernel(T* __restrict__ buf, int ld, int ncols, int planes, long long plane_ld,
                                 const int* __restrict__ start, int nrows, int max_rows) {
  const long long r0 = *start;
  const long long r1 = min((long long)max_rows, r0 + nrows);
  if (r1 <= r0) return;
  const long long per_plane = (r1 - r0) * ncols;
  const long long total = per_plane * planes;
  for (long long w = (long long)blockIdx.x * blockDim.x + threadIdx.x; w < total;
       w += (long long)gridDim.x * blockDim.x) {
    const long long p = w / per_plane, rem = w - p * per_plane;
    const long long r = r0 + rem / ncols, c = rem % ncols;
    buf[p * plane_ld + r * ld + c] = from_f<T>(0.f);
  }
}

template <typename T>
cudaError_t launch_zero_rows(T* buf, int ld, int ncols, int planes, long long plane_ld, const int* start, int nrows,
                             int max_rows, cudaStream_t st) {
  const int grid = grid_for((long long)nrows * ncols * planes, 256, device_sm_count() * 4);
  zero_rows_kernel<T><<<grid, 256, 0, st>>>(buf, ld, ncols, planes, plane_ld, start, nrows, max_rows);
  return cudaGetLastError();
}

// -------------------------------------------------------------------- SwiGLU
__device__ __forceinline__ float sigmoidf_(float g) { return 1.0f / (1.0f + expf(-g)); }

// h = silu(g) * u with g = gu[:, j], u = gu[:, F + j]; 8 columns per thread.
template <typename T>
__global__ void swiglu_fwd_kernel(const T* __restrict__ gu, T* __restrict__ h, const int* __restrict__ cnt, int S,
                                  int F) {
  const long long M = (long long)(*cnt) * S;
  const int F8 = F / 8;
  const long long total = M * F8;
  for (long long w = (long long)blockIdx.x * blockDim.x + threadIdx.x; w < total;
       w += (long long)gridDim.x * blockDim.x) {
    const long long m = w / F8;
    const int j = (int)(w - m * F8) * 8;
    float g[8], u[8], o[8];
    ld8(gu + m * 2 * F + j, g);
    ld8(gu + m * 2 * F + F + j, u);
#pragma unroll
    for (int k = 0; k < 8; ++k) o[k] = g[k] * sigmoidf_(g[k]) * u[k];
    st8(h + m * F + j, o);
  }
}

template <typename T>
cudaError_t launch_swiglu_fwd(const T* gu, T* h, const int* cnt, int S, int F, int max_rows, cudaStream_t st) {
  const int grid = grid_for((long long)max_rows * (F / 8), 256, device_sm_count() * 8);
  swiglu_fwd_kernel<T><<<grid, 256, 0, st>>>(gu, h, cnt, S, F);
  return cudaGetLastError();
}

// dg = dh * u * s (1 + g (1 - s)), du = dh * g * s with s = sigmoid(g).
template <typename T>
__global__ void swiglu_bwd_kernel(const T* __restrict__ dh, const T* __restrict__ gu, T* __restrict__ dgu,
                                  const int* __restrict__ cnt, int S, int F) {
  const long long M = (long long)(*cnt) * S;
  const int F8 = F / 8;
  const long long total = M * F8;
  for (long long w = (long long)blockIdx.x * blockDim.x + threadIdx.x; w < total;
       w += (long long)gridDim.x * blockDim.x) {
    const long long m = w / F8;
    const int j = (int)(w - m * F8) * 8;
    float g[8], u[8], dv[8], dg[8], du[8];
    ld8(gu + m * 2 * F + j, g);
    ld8(gu + m * 2 * F + F + j, u);
    ld8(dh + m * F + j, dv);
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const float sg = sigmoidf_(g[k]);
      dg[k] = dv[k] * u[k] * sg * (1.0f + g[k] * (1.0f - sg));
      du[k] = dv[k] * g[k] * sg;
    }
    st8(dgu + m * 2 * F + j, dg);
    st8(dgu + m * 2 * F + F + j, du);
  }
}

template <typename T>
cudaError_t launch_swiglu_bwd(const T* dh, const T* gu, T* dgu, const int* cnt, int S, int F, int max_rows,
                              cudaStream_t st) {
  const int grid = grid_for((long long)max_rows * (F / 8), 256, device_sm_count() * 8);
  swiglu_bwd_kernel<T><<<grid, 256, 0, st>>>(dh, gu, dgu, cnt, S, F);
  return cudaGetLastError();
}

// ------------------------------------------------------------ ALiBi slopes
// Press et al., "Train Short, Test Long" (ICLR 2022): with n0 the largest
// power of two <= H, head h < n0 has slope 2^(-8 (h + 1) / n0); head
// n0 + k has 2^(-4 (2k + 1) / n0), every other slope of the 2 n0 sequence.
__global__ void alibi_table_kernel(float* __restrict__ slopes, int H) {
  int n0 = 1;
  while (n0 * 2 <= H) n0 *= 2;
  for (int h = threadIdx.x; h < H; h += blockDim.x) {
    const double e = h < n0 ? -8.0 * (h + 1) / n0 : -4.0 * (2 * (h - n0) + 1) / n0;
    slopes[h] = (float)exp2(e);
  }
}

cudaError_t launch_alibi_table(float* slopes, int H, cudaStream_t st) {
  alibi_table_kernel<<<1, 256, 0, st>>>(slopes, H);
  return cudaGetLastError();
}

// ------------------------------------------------------------ squared ReLU
// h = max(u, 0)^2 (forward); du = dh * 2 max(u, 0) (backward); [M, F] rows.
template <typename T>
__global__ void relu2_kernel(const T* __restrict__ u, const T* __restrict__ dh, T* __restrict__ out,
                             const int* __restrict__ cnt, int S, int F) {
  const long long total = (long long)(*cnt) * S * (F / 8);
  for (long long w = (long long)blockIdx.x * blockDim.x + threadIdx.x; w < total;
       w += (long long)gridDim.x * blockDim.x) {
    float uv[8], o[8];
    ld8(u + w * 8, uv);
    if (dh) {
      float dv[8];
      ld8(dh + w * 8, dv);
#pragma unroll
      for (int k = 0; k < 8; ++k) o[k] = dv[k] * 2.f * fmaxf(uv[k], 0.f);
    } else {
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const float r = fmaxf(uv[k], 0.f);
        o[k] = r * r;
      }
    }
    st8(out + w * 8, o);
  }
}

template <typename T>
cudaError_t launch_relu2(const T* u, const T* dh, T* out, const int* cnt, int S, int F, int max_rows,
                         cudaStream_t st) {
  const int grid = grid_for((long long)max_rows * (F / 8), 256, device_sm_count() * 8);
  relu2_kernel<T><<<grid, 256, 0, st>>>(u, dh, out, cnt, S, F);
  return cudaGetLastError();
}

// ------------------------------------------- attention backward preprocess
// Dvec[h][m] = sum_i dO[m, h*Dh+i] * O[m, h*Dh+i]  (row sum of dP * P).
template <typename T>
__global__ void attn_rowdot_kernel(const T* __restrict__ dO, const T* __restrict__ O, int ld, int H, int Dh,
                                   const int* __restrict__ cnt, int S, int max_rows, float* __restrict__ Dvec) {
  // one warp per row, all heads: lane l takes elements 8l + 256k of the row
  // (16-byte loads), the Dh / 8 lanes of a head sum their dot products with
  // shuffles, and the head's first lane stores it
  const long long M = (long long)(*cnt) * S;
  const int lane = threadIdx.x & 31;
  const int HD = H * Dh, G = Dh / 8;  // lanes per head within a 256-element block
  const long long nwarps = (long long)gridDim.x * (blockDim.x >> 5);
  for (long long m = (long long)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); m < M; m += nwarps) {
    const T* a = dO + m * ld;
    const T* b = O + m * ld;
    for (int i0 = 0; i0 < HD; i0 += 256) {
      const int i = i0 + lane * 8;
      float s = 0.f;
      if (i < HD) {
        float x[8], y[8];
        ld8(a + i, x);
        ld8(b + i, y);
#pragma unroll
        for (int e = 0; e < 8; ++e) s += x[e] * y[e];
      }
      for (int off = G >> 1; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
      if (i < HD && (lane % G) == 0) Dvec[(size_t)(i / Dh) * max_rows + m] = s;
    }
  }
}

template <typename T>
cudaError_t launch_attn_rowdot(const T* dO, const T* O, int ld, int H, int Dh, const int* cnt, int S, int max_rows,
                               float* Dvec, cudaStream_t st) {
  if (Dh < 8 || Dh > 256 || (Dh & (Dh - 1))) return cudaErrorInvalidValue;  // head groups of Dh / 8 lanes
  const int grid = grid_for((long long)max_rows, 8, device_sm_count() * 16);
  attn_rowdot_kernel<T><<<grid, 256, 0, st>>>(dO, O, ld, H, Dh, cnt, S, max_rows, Dvec);
  return cudaGetLastError();
}

#define LD_INST(T)                                                                                              \
  template cudaError_t launch_rmsnorm_fwd<float, T>(const float*, int, const int*, const int*, int, int, int,   \
                                                    const T*, float, float*, T*, float*, cudaStream_t);         \
  template cudaError_t launch_rmsnorm_bwd<T>(const float*, const float*, const float*, const T*, float*,         \
                                             const int*,                                                         \
                                             const int*, int, int, int, float, T*, float*, int, cudaStream_t);  \
  template cudaError_t launch_gather_scale<T>(const float*, const int*, const int*, int, int, int, float, T*,    \
                                              cudaStream_t);                                                    \
  template cudaError_t launch_rope_apply<T>(T*, int, int, int, const float*, const float*, const int*, int, int, \
                                            int, const int*, cudaStream_t);                                     \
  template cudaError_t launch_zero_rows<T>(T*, int, int, int, long long, const int*, int, int, cudaStream_t);   \
  template cudaError_t launch_swiglu_fwd<T>(const T*, T*, const int*, int, int, int, cudaStream_t);             \
  template cudaError_t launch_swiglu_bwd<T>(const T*, const T*, T*, const int*, int, int, int, cudaStream_t);   \
  template cudaError_t launch_relu2<T>(const T*, const T*, T*, const int*, int, int, int, cudaStream_t);        \
  template cudaError_t launch_attn_rowdot<T>(const T*, const T*, int, int, int, const int*, int, int, float*,   \
                                             cudaStream_t);
LD_INST(bf16)
template cudaError_t launch_rmsnorm_fwd<float, float>(const float*, int, const int*, const int*, int, int, int,
                                                      const float*, float, float*, float*, float*, cudaStream_t);
template cudaError_t launch_rmsnorm_bwd<float>(const float*, const float*, const float*, const float*, float*,
                                               const int*, const int*, int, int, int, float, float*, float*, int,
                                               cudaStream_t);
template cudaError_t launch_gather_scale<float>(const float*, const int*, const int*, int, int, int, float, float*,
                                                cudaStream_t);
template cudaError_t launch_rope_apply<float>(float*, int, int, int, const float*, const float*, const int*, int, int,
                                              int, const int*, cudaStream_t);
template cudaError_t launch_zero_rows<float>(float*, int, int, int, long long, const int*, int, int, cudaStream_t);
template cudaError_t launch_swiglu_fwd<float>(const float*, float*, const int*, int, int, int, cudaStream_t);
template cudaError_t launch_swiglu_bwd<float>(const float*, const float*, float*, const int*, int, int, int,
                                              cudaStream_t);
template cudaError_t launch_relu2<float>(const float*, const float*, float*, const int*, int, int, int, cudaStream_t);
template cudaError_t launch_attn_rowdot<float>(const float*, const float*, int, int, int, const int*, int, int,
                                               float*, cudaStream_t);

}  // namespace ldk
