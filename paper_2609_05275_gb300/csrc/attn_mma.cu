// Causal grouped-query flash attention for bf16 on tensor cores
// (mma.sync m16n8k16, fp32 accumulation), forward and backward.
//
// f_attn of Eq. (transformer_layer_dropout_train), per kept sequence s and
// query head h (key/value head g = floor(h*Hkv/H)):
//   o_i = sum_{j<=i} softmax_j(c q_i . k_j [+ m_h (j - i)]) v_j,   c = 1/sqrt(Dh)
// (the bracket with an ALiBi slope table, m_h per query head).
// Rows are compact: kept sequence s occupies rows s*S .. s*S+S-1 of qkv
// ([Q heads | K heads | V heads] columns).  The grid covers every batch slot
// and blocks past the layer's kept count return at once, so the launch is
// independent of the mask.
//
// Forward: one CTA per (64-query tile, head, sequence), online softmax in
// base 2, K/V tiles double-buffered with cp.async; writes o and the
// log-sum-exp (natural log) per (head, row).
// Backward: one CTA per (64-key tile, kv head, sequence) loops over the
// query heads of its group and the query tiles at or after its key tile,
// recomputes P from the saved log-sum-exp, accumulates dK and dV in
// registers (summed over the group, as GQA shares them) and adds dQ into a
// float32 buffer with atomics; dq_finish scales it into dqkv.
#include "ld_internal.cuh"

namespace ldk {
namespace {

__device__ __forceinline__ uint32_t saddr(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void cp16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(saddr(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

__device__ __forceinline__ void ldsm4(uint32_t a, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(a));
}
__device__ __forceinline__ void ldsm4t(uint32_t a, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(a));
}
// D += A (16x16, row) * B (16x8, col), bf16 inputs, fp32 accumulator.
__device__ __forceinline__ void mma(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t pack(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

// Copy a [64 x DH] tile (global row stride ld) into shared [64][DH+8].
template <int DH>
__device__ __forceinline__ void load_tile(bf16* dst, const bf16* src, long long ld, int tid) {
  constexpr int CPR = DH / 8, LDS = DH + 8;
#pragma unroll 4
  for (int i = tid; i < 64 * CPR; i += 128) {
    const int r = i / CPR, c = (i % CPR) * 8;
    cp16(dst + r * LDS + c, src + (long long)r * ld + c);
  }
}

// A fragment (16 x 16) at (row0, col0) of a row-major shared matrix.
__device__ __forceinline__ void frag_a(const bf16* base, int ld, int row0, int col0, int lane, uint32_t (&a)[4]) {
  ldsm4(saddr(base + (row0 + (lane & 15)) * ld + col0 + (lane >> 4) * 8), a[0], a[1], a[2], a[3]);
}
// B fragments of two n-tiles (n0..n0+15) x k0..k0+15 from shared [n][k].
__device__ __forceinline__ void frag_b_nk(const bf16* base, int ld, int n0, int k0, int lane, uint32_t& b0,
                                          uint32_t& b1, uint32_t& b2, uint32_t& b3) {
  ldsm4(saddr(base + (n0 + (lane & 7) + ((lane >> 4) << 3)) * ld + k0 + ((lane >> 3) & 1) * 8), b0, b1, b2, b3);
}
// B fragments of two n-tiles (n0..n0+15) x k0..k0+15 from shared [k][n].
__device__ __forceinline__ void frag_b_kn(const bf16* base, int ld, int k0, int n0, int lane, uint32_t& b0,
                                          uint32_t& b1, uint32_t& b2, uint32_t& b3) {
  ldsm4t(saddr(base + (k0 + (lane & 7) + (((lane >> 3) & 1) << 3)) * ld + n0 + (lane >> 4) * 8), b0, b1, b2, b3);
}

template <int DH>
__global__ void __launch_bounds__(128) attn_fwd_kernel(const bf16* __restrict__ qkv, int ldq, bf16* __restrict__ o,
                                                       int ldo, float* __restrict__ lse, int lse_ld,
                                                       const int* __restrict__ cnt, int S, int H, int Hkv,
                                                       const float* __restrict__ alibi) {
  constexpr int LDS = DH + 8, NDT = DH / 8, NKC = DH / 16;
  extern __shared__ __align__(16) uint8_t smraw[];
  bf16* Qs = reinterpret_cast<bf16*>(smraw);
  bf16* Ks = Qs + 64 * LDS;
  bf16* Vs = Ks + 2 * 64 * LDS;
  const int seq = blockIdx.z;
  if (seq >= *cnt) return;
  const int nqt = S / 64;
  const int qt = nqt - 1 - blockIdx.x;  // heaviest tiles first
  const int h = blockIdx.y, g = (h * Hkv) / H;
  const long long row0 = (long long)seq * S;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const bf16* Kg = qkv + row0 * ldq + (long long)(H + g) * DH;
  const bf16* Vg = qkv + row0 * ldq + (long long)(H + Hkv + g) * DH;

  load_tile<DH>(Qs, qkv + (row0 + qt * 64) * ldq + (long long)h * DH, ldq, tid);
  load_tile<DH>(Ks, Kg, ldq, tid);
  load_tile<DH>(Vs, Vg, ldq, tid);
  cp_commit();
  cp_wait<0>();
  __syncthreads();
  uint32_t qf[NKC][4];
#pragma unroll
  for (int kc = 0; kc < NKC; ++kc) frag_a(Qs, LDS, warp * 16, kc * 16, lane, qf[kc]);

  float oacc[NDT][4];
#pragma unroll
  for (int i = 0; i < NDT; ++i) oacc[i][0] = oacc[i][1] = oacc[i][2] = oacc[i][3] = 0.f;
  float mrow[2] = {-INFINITY, -INFINITY}, lrow[2] = {0.f, 0.f};
  const float sl2 = rsqrtf((float)DH) * kLog2e;
  const float slope2 = alibi ? alibi[h] * kLog2e : 0.f;  // ALiBi bias slope2 (key - query), base 2
  const int qr0 = qt * 64 + warp * 16 + (lane >> 2);  // this thread's rows: qr0, qr0 + 8

  for (int kt = 0; kt <= qt; ++kt) {
    const int buf = kt & 1;
    if (kt + 1 <= qt) {
      load_tile<DH>(Ks + (buf ^ 1) * 64 * LDS, Kg + (long long)(kt + 1) * 64 * ldq, ldq, tid);
      load_tile<DH>(Vs + (buf ^ 1) * 64 * LDS, Vg + (long long)(kt + 1) * 64 * ldq, ldq, tid);
    }
    cp_commit();
    cp_wait<1>();
    __syncthreads();
    const bf16* K_ = Ks + buf * 64 * LDS;
    const bf16* V_ = Vs + buf * 64 * LDS;
    float s[8][4];
#pragma unroll
    for (int i = 0; i < 8; ++i) s[i][0] = s[i][1] = s[i][2] = s[i][3] = 0.f;
#pragma unroll
    for (int kc = 0; kc < NKC; ++kc) {
#pragma unroll
      for (int np = 0; np < 4; ++np) {
        uint32_t b0, b1, b2, b3;
        frag_b_nk(K_, LDS, np * 16, kc * 16, lane, b0, b1, b2, b3);
        mma(s[2 * np], qf[kc], b0, b1);
        mma(s[2 * np + 1], qf[kc], b2, b3);
      }
    }
    float mx[2] = {mrow[0], mrow[1]};
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int key = kt * 64 + nt * 8 + 2 * (lane & 3) + (e & 1);
        const int qr = qr0 + (e >> 1) * 8;
        float v = fmaf(s[nt][e], sl2, slope2 * (float)(key - qr));
        if (kt == qt && key > qr) v = -INFINITY;
        s[nt][e] = v;
        mx[e >> 1] = fmaxf(mx[e >> 1], v);
      }
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 1));
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 2));
    }
    const float corr0 = exp2f(mrow[0] - mx[0]), corr1 = exp2f(mrow[1] - mx[1]);
    mrow[0] = mx[0];
    mrow[1] = mx[1];
    float ls0 = 0.f, ls1 = 0.f;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      s[nt][0] = exp2f(s[nt][0] - mx[0]);
      s[nt][1] = exp2f(s[nt][1] - mx[0]);
      s[nt][2] = exp2f(s[nt][2] - mx[1]);
      s[nt][3] = exp2f(s[nt][3] - mx[1]);
      ls0 += s[nt][0] + s[nt][1];
      ls1 += s[nt][2] + s[nt][3];
    }
    lrow[0] = lrow[0] * corr0 + ls0;
    lrow[1] = lrow[1] * corr1 + ls1;
#pragma unroll
    for (int dt = 0; dt < NDT; ++dt) {
      oacc[dt][0] *= corr0;
      oacc[dt][1] *= corr0;
      oacc[dt][2] *= corr1;
      oacc[dt][3] *= corr1;
    }
#pragma unroll
    for (int kc = 0; kc < 4; ++kc) {
      uint32_t pa[4] = {pack(s[2 * kc][0], s[2 * kc][1]), pack(s[2 * kc][2], s[2 * kc][3]),
                        pack(s[2 * kc + 1][0], s[2 * kc + 1][1]), pack(s[2 * kc + 1][2], s[2 * kc + 1][3])};
#pragma unroll
      for (int dp = 0; dp < NDT / 2; ++dp) {
        uint32_t b0, b1, b2, b3;
        frag_b_kn(V_, LDS, kc * 16, dp * 16, lane, b0, b1, b2, b3);
        mma(oacc[2 * dp], pa, b0, b1);
        mma(oacc[2 * dp + 1], pa, b2, b3);
      }
    }
    __syncthreads();
  }
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 1);
    lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 2);
  }
  const float inv0 = 1.0f / lrow[0], inv1 = 1.0f / lrow[1];
  bf16* o0 = o + (row0 + qr0) * ldo + (long long)h * DH + 2 * (lane & 3);
  bf16* o1 = o0 + 8LL * ldo;
#pragma unroll
  for (int dt = 0; dt < NDT; ++dt) {
    *reinterpret_cast<uint32_t*>(o0 + dt * 8) = pack(oacc[dt][0] * inv0, oacc[dt][1] * inv0);
    *reinterpret_cast<uint32_t*>(o1 + dt * 8) = pack(oacc[dt][2] * inv1, oacc[dt][3] * inv1);
  }
  if ((lane & 3) == 0) {
    lse[(size_t)h * lse_ld + row0 + qr0] = (mrow[0] + log2f(lrow[0])) * kLn2;
    lse[(size_t)h * lse_ld + row0 + qr0 + 8] = (mrow[1] + log2f(lrow[1])) * kLn2;
  }
}

template <int DH>
__global__ void __launch_bounds__(128) attn_bwd_kernel(const bf16* __restrict__ qkv, int ldq,
                                                       const bf16* __restrict__ dO, int ldo,
                                                       const float* __restrict__ lse, const float* __restrict__ Dvec,
                                                       int lse_ld, float* __restrict__ dq_acc,
                                                       bf16* __restrict__ dqkv, const int* __restrict__ cnt, int S,
                                                       int H, int Hkv, const float* __restrict__ alibi) {
  constexpr int LDS = DH + 8, NDT = DH / 8, NKC = DH / 16, LDP = 64 + 8;
  extern __shared__ __align__(16) uint8_t smraw[];
  bf16* Ks = reinterpret_cast<bf16*>(smraw);
  bf16* Vs = Ks + 64 * LDS;
  bf16* Qs = Vs + 64 * LDS;
  bf16* dOs = Qs + 64 * LDS;
  bf16* dSs = dOs + 64 * LDS;  // [64 queries][64 keys]
  float* lse_s = reinterpret_cast<float*>(dSs + 64 * LDP);
  float* D_s = lse_s + 64;
  const int seq = blockIdx.z;
  if (seq >= *cnt) return;
  const int nqt = S / 64;
  const int kt = blockIdx.x;
  const int g = blockIdx.y, grp = H / Hkv;
  const long long row0 = (long long)seq * S;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int HD = H * DH;

  load_tile<DH>(Ks, qkv + (row0 + kt * 64) * ldq + (long long)(H + g) * DH, ldq, tid);
  load_tile<DH>(Vs, qkv + (row0 + kt * 64) * ldq + (long long)(H + Hkv + g) * DH, ldq, tid);
  cp_commit();

  float dk[NDT][4], dv[NDT][4];
#pragma unroll
  for (int i = 0; i < NDT; ++i)
#pragma unroll
    for (int e = 0; e < 4; ++e) dk[i][e] = dv[i][e] = 0.f;
  const float sl2 = rsqrtf((float)DH) * kLog2e;
  const int kr0 = kt * 64 + warp * 16 + (lane >> 2);  // this thread's keys: kr0, kr0 + 8

  for (int h = g * grp; h < (g + 1) * grp; ++h) {
    const float slope2 = alibi ? alibi[h] * kLog2e : 0.f;
    for (int qt = kt; qt < nqt; ++qt) {
      const long long qrow = row0 + qt * 64;
      load_tile<DH>(Qs, qkv + qrow * ldq + (long long)h * DH, ldq, tid);
      load_tile<DH>(dOs, dO + qrow * ldo + (long long)h * DH, ldo, tid);
      cp_commit();
      if (tid < 64) {
        lse_s[tid] = lse[(size_t)h * lse_ld + qrow + tid] * kLog2e;
        D_s[tid] = Dvec[(size_t)h * lse_ld + qrow + tid];
      }
      cp_wait<0>();
      __syncthreads();
      // S^T and dP^T for this warp's 16 keys x 64 queries
      float st[8][4], dp[8][4];
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int e = 0; e < 4; ++e) st[i][e] = dp[i][e] = 0.f;
#pragma unroll
      for (int kc = 0; kc < NKC; ++kc) {
        uint32_t ka[4], va[4];
        frag_a(Ks, LDS, warp * 16, kc * 16, lane, ka);
        frag_a(Vs, LDS, warp * 16, kc * 16, lane, va);
#pragma unroll
        for (int np = 0; np < 4; ++np) {
          uint32_t b0, b1, b2, b3;
          frag_b_nk(Qs, LDS, np * 16, kc * 16, lane, b0, b1, b2, b3);
          mma(st[2 * np], ka, b0, b1);
          mma(st[2 * np + 1], ka, b2, b3);
          frag_b_nk(dOs, LDS, np * 16, kc * 16, lane, b0, b1, b2, b3);
          mma(dp[2 * np], va, b0, b1);
          mma(dp[2 * np + 1], va, b2, b3);
        }
      }
      // P^T (into st) and dS^T (into dp)
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int ql = nt * 8 + 2 * (lane & 3) + (e & 1);
          const int key = kr0 + (e >> 1) * 8;
          const float x = fmaf(st[nt][e], sl2, slope2 * (float)(key - qt * 64 - ql));
          const float p = (qt * 64 + ql >= key) ? exp2f(x - lse_s[ql]) : 0.f;
          st[nt][e] = p;
          dp[nt][e] = p * (dp[nt][e] - D_s[ql]);
        }
      }
      // dV += P^T dO ; dK += dS^T Q   (contraction over the 64 queries)
#pragma unroll
      for (int kc = 0; kc < 4; ++kc) {
        uint32_t pa[4] = {pack(st[2 * kc][0], st[2 * kc][1]), pack(st[2 * kc][2], st[2 * kc][3]),
                          pack(st[2 * kc + 1][0], st[2 * kc + 1][1]), pack(st[2 * kc + 1][2], st[2 * kc + 1][3])};
        uint32_t sa[4] = {pack(dp[2 * kc][0], dp[2 * kc][1]), pack(dp[2 * kc][2], dp[2 * kc][3]),
                          pack(dp[2 * kc + 1][0], dp[2 * kc + 1][1]), pack(dp[2 * kc + 1][2], dp[2 * kc + 1][3])};
#pragma unroll
        for (int dq2 = 0; dq2 < NDT / 2; ++dq2) {
          uint32_t b0, b1, b2, b3;
          frag_b_kn(dOs, LDS, kc * 16, dq2 * 16, lane, b0, b1, b2, b3);
          mma(dv[2 * dq2], pa, b0, b1);
          mma(dv[2 * dq2 + 1], pa, b2, b3);
          frag_b_kn(Qs, LDS, kc * 16, dq2 * 16, lane, b0, b1, b2, b3);
          mma(dk[2 * dq2], sa, b0, b1);
          mma(dk[2 * dq2 + 1], sa, b2, b3);
        }
      }
      // dS as [query][key] in shared memory for dQ = dS K
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int ql = nt * 8 + 2 * (lane & 3) + (e & 1);
          const int kl = warp * 16 + (lane >> 2) + (e >> 1) * 8;
          dSs[ql * LDP + kl] = __float2bfloat16_rn(dp[nt][e]);
        }
      }
      __syncthreads();
      // dQ rows 16*warp .. +15 of this query tile, in column chunks of 32
      float* dqrow0 = dq_acc + (qrow + warp * 16 + (lane >> 2)) * (long long)HD + (long long)h * DH + 2 * (lane & 3);
#pragma unroll
      for (int cc = 0; cc < DH / 32; ++cc) {
        float acc[4][4];
#pragma unroll
        for (int i = 0; i < 4; ++i) acc[i][0] = acc[i][1] = acc[i][2] = acc[i][3] = 0.f;
#pragma unroll
        for (int kc = 0; kc < 4; ++kc) {
          uint32_t a[4];
          frag_a(dSs, LDP, warp * 16, kc * 16, lane, a);
#pragma unroll
          for (int np = 0; np < 2; ++np) {
            uint32_t b0, b1, b2, b3;
            frag_b_kn(Ks, LDS, kc * 16, cc * 32 + np * 16, lane, b0, b1, b2, b3);
            mma(acc[2 * np], a, b0, b1);
            mma(acc[2 * np + 1], a, b2, b3);
          }
        }
#pragma unroll
        for (int nt = 0; nt < 4; ++nt) {
          float* p0 = dqrow0 + cc * 32 + nt * 8;
          atomicAdd(p0, acc[nt][0]);
          atomicAdd(p0 + 1, acc[nt][1]);
          atomicAdd(p0 + 8LL * HD, acc[nt][2]);
          atomicAdd(p0 + 8LL * HD + 1, acc[nt][3]);
        }
      }
      __syncthreads();
    }
  }
  // dK (times c) and dV for this key tile
  const float c = rsqrtf((float)DH);
  bf16* k0 = dqkv + (row0 + kr0) * ldq + (long long)(H + g) * DH + 2 * (lane & 3);
  bf16* v0 = dqkv + (row0 + kr0) * ldq + (long long)(H + Hkv + g) * DH + 2 * (lane & 3);
#pragma unroll
  for (int dt = 0; dt < NDT; ++dt) {
    *reinterpret_cast<uint32_t*>(k0 + dt * 8) = pack(c * dk[dt][0], c * dk[dt][1]);
    *reinterpret_cast<uint32_t*>(k0 + 8LL * ldq + dt * 8) = pack(c * dk[dt][2], c * dk[dt][3]);
    *reinterpret_cast<uint32_t*>(v0 + dt * 8) = pack(dv[dt][0], dv[dt][1]);
    *reinterpret_cast<uint32_t*>(v0 + 8LL * ldq + dt * 8) = pack(dv[dt][2], dv[dt][3]);
  }
}

// dq = c * dq_acc, then the inverse rotary rotation of each q head (pairs
// (i, i + Dh/2) at the row's position), written as bf16 into dqkv.
__global__ void dq_finish_kernel(const float* __restrict__ dq_acc, bf16* __restrict__ dqkv, int ldq, int H, int Dh,
                                 float c, const float* __restrict__ rcos, const float* __restrict__ rsin,
                                 const int* __restrict__ cnt, int S, const int* __restrict__ tok) {
  const long long M = tok ? (long long)(*cnt) : (long long)(*cnt) * S;
  const int half = Dh / 2, HD = H * Dh;
  const int per_row = H * (half / 4);
  const long long total = M * per_row;
  for (long long w = (long long)blockIdx.x * blockDim.x + threadIdx.x; w < total;
       w += (long long)gridDim.x * blockDim.x) {
    const long long m = w / per_row;
    const int rem = (int)(w - m * per_row);
    const int h = rem / (half / 4), i = (rem - h * (half / 4)) * 4;
    const float* src = dq_acc + m * HD + (long long)h * Dh + i;
    const float4 a = *reinterpret_cast<const float4*>(src);
    const float4 b = *reinterpret_cast<const float4*>(src + half);
    float x1[4] = {c * a.x, c * a.y, c * a.z, c * a.w}, x2[4] = {c * b.x, c * b.y, c * b.z, c * b.w};
    if (rcos) {
      const int pos = row_pos(tok, S, m);
      const float4 cv = *reinterpret_cast<const float4*>(rcos + (size_t)pos * half + i);
      const float4 sv = *reinterpret_cast<const float4*>(rsin + (size_t)pos * half + i);
      const float cs[4] = {cv.x, cv.y, cv.z, cv.w}, sn[4] = {sv.x, sv.y, sv.z, sv.w};
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const float p1 = x1[k], p2 = x2[k];
        x1[k] = p1 * cs[k] + p2 * sn[k];
        x2[k] = p2 * cs[k] - p1 * sn[k];
      }
    }
    bf16* dst = dqkv + m * ldq + (long long)h * Dh + i;
    uint2 o1, o2;
    o1.x = pack(x1[0], x1[1]);
    o1.y = pack(x1[2], x1[3]);
    o2.x = pack(x2[0], x2[1]);
    o2.y = pack(x2[2], x2[3]);
    *reinterpret_cast<uint2*>(dst) = o1;
    *reinterpret_cast<uint2*>(dst + half) = o2;
  }
}

template <int DH>
cudaError_t fwd_launch(const bf16* qkv, int ldq, bf16* o, int ldo, float* lse, const int* cnt, int S, int H, int Hkv,
                       int max_seqs, const float* alibi, cudaStream_t st) {
  constexpr size_t smem = (size_t)5 * 64 * (DH + 8) * sizeof(bf16);
  // once per process (initialisation of a function-local static is thread-safe)
  static const cudaError_t attr =
      cudaFuncSetAttribute(attn_fwd_kernel<DH>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (attr != cudaSuccess) return attr;
  dim3 grid(S / 64, H, max_seqs);
  attn_fwd_kernel<DH><<<grid, 128, smem, st>>>(qkv, ldq, o, ldo, lse, max_seqs * S, cnt, S, H, Hkv, alibi);
  return cudaGetLastError();
}

template <int DH>
cudaError_t bwd_launch(const bf16* qkv, int ldq, const bf16* dO, int ldo, const float* lse, const float* Dvec,
                       float* dq_acc, bf16* dqkv, const int* cnt, int S, int H, int Hkv, int max_seqs,
                       const float* alibi, cudaStream_t st) {
  constexpr size_t smem = (size_t)4 * 64 * (DH + 8) * sizeof(bf16) + 64 * 72 * sizeof(bf16) + 128 * sizeof(float);
  // once per process (initialisation of a function-local static is thread-safe)
  static const cudaError_t attr =
      cudaFuncSetAttribute(attn_bwd_kernel<DH>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (attr != cudaSuccess) return attr;
  dim3 grid(S / 64, Hkv, max_seqs);
  attn_bwd_kernel<DH><<<grid, 128, smem, st>>>(qkv, ldq, dO, ldo, lse, Dvec, max_seqs * S, dq_acc, dqkv, cnt, S, H,
                                               Hkv, alibi);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_attn_fwd_mma(const bf16* qkv, int ldqkv, bf16* o, int ldo, float* lse, const int* cnt, int S, int H,
                                int Hkv, int Dh, int max_seqs, const float* alibi, cudaStream_t st) {
  if (Dh == 32) return fwd_launch<32>(qkv, ldqkv, o, ldo, lse, cnt, S, H, Hkv, max_seqs, alibi, st);
  if (Dh == 64) return fwd_launch<64>(qkv, ldqkv, o, ldo, lse, cnt, S, H, Hkv, max_seqs, alibi, st);
  return fwd_launch<128>(qkv, ldqkv, o, ldo, lse, cnt, S, H, Hkv, max_seqs, alibi, st);
}

cudaError_t launch_attn_bwd_mma(const bf16* qkv, int ldqkv, const bf16* o, const bf16* dO, int ldo, const float* lse,
                                const float* Dvec, float* dq_acc, bf16* dqkv, const int* cnt, int S, int H, int Hkv,
                                int Dh, int max_seqs, const float* alibi, cudaStream_t st) {
  (void)o;
  cudaError_t e = cudaMemsetAsync(dq_acc, 0, (size_t)max_seqs * S * H * Dh * sizeof(float), st);
  if (e != cudaSuccess) return e;
  if (Dh == 32) return bwd_launch<32>(qkv, ldqkv, dO, ldo, lse, Dvec, dq_acc, dqkv, cnt, S, H, Hkv, max_seqs, alibi, st);
  if (Dh == 64) return bwd_launch<64>(qkv, ldqkv, dO, ldo, lse, Dvec, dq_acc, dqkv, cnt, S, H, Hkv, max_seqs, alibi, st);
  return bwd_launch<128>(qkv, ldqkv, dO, ldo, lse, Dvec, dq_acc, dqkv, cnt, S, H, Hkv, max_seqs, alibi, st);
}

cudaError_t launch_dq_finish(const float* dq_acc, bf16* dqkv, int ldqkv, int H, int Dh, const float* rcos,
                             const float* rsin, const int* cnt, int S, int max_rows, const int* tok, cudaStream_t st) {
  long long work = (long long)max_rows * H * (Dh / 8);
  long long grid = (work + 255) / 256;
  const long long cap = (long long)device_sm_count() * 8;
  if (grid > cap) grid = cap;
  if (grid < 1) grid = 1;
  dq_finish_kernel<<<(int)grid, 256, 0, st>>>(dq_acc, dqkv, ldqkv, H, Dh, rsqrtf((float)Dh), rcos, rsin, cnt, S, tok);
  return cudaGetLastError();
}

}  // namespace ldk
