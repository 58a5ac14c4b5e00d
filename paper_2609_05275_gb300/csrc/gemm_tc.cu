// bf16 GEMM on the 5th-generation tensor cores (tcgen05) for sm_103a:
//   D(m,n) = alpha * sum_k A(m,k) B(n,k)   (fp32 accumulation in TMEM)
//
// These are the dense contractions of the block (the projections inside
// f_attn and f_ffn of Eq. (transformer_layer_dropout_train)) and their
// gradients, run only on the kept rows: the row extent M (forward and
// data-gradient products) or the contraction extent K (weight-gradient
// products) is read from the layer's kept count in device memory, so the
// work shrinks with the number of kept sequences without a host round trip.
//
// Structure (persistent, one CTA per SM, 192 threads):
//   warp 0      TMA producer: 128B-swizzled tiles of A (128 x 64) and
//               B (BN x 64) into a STAGES-deep shared-memory ring whose
//               stages hold KPS such k-blocks (one barrier hand-off each);
//   warp 1      allocates 2*BN TMEM columns (two accumulators) and issues
//               tcgen05.mma (M=128, N=BN, K=16) from one thread;
//   warps 2..5  epilogue: tcgen05.ld of the accumulator (each warp reads
//               its 32-lane quadrant), fused scale / residual update, and
//               global stores, overlapped with the next tile's MMAs.
// 256-column tiles run on CTA pairs (clusters of two on the SMs of a TPC):
// a 256 x 256 tile per pair, each CTA loading 128 rows of A and 128 rows of
// B, one tcgen05.mma.cta_group::2 (M=256) per K=16 step from the even CTA.
// Operands may be K-major or MN-major (weight-gradient and data-gradient
// products read activations and weights transposed); the shared-memory
// descriptors and the instruction descriptor's major bits cover both, so no
// transpose is ever materialised.
//
// Every mbarrier wait is bounded: after kWaitLimitNs the CTA raises the
// status word (LD_ERR_TIMEOUT), drains its own TMA copies and MMAs with a
// further bounded wait, frees its TMEM and exits (a CTA pair meets at a
// cluster barrier first, so neither frees memory the other may address).
// Per-token kept lists pass padding rows (kept index -1): the residual
// epilogue skips them and writes zeros to its compact copy.
#include <cuda.h>
#include <cudaTypedefs.h>

#include "tc_common.cuh"

namespace ldk {
namespace tc {
// ---------------------------------------------------------------- host side
static PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  // once per process (initialisation of a function-local static is thread-safe)
  static const PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    return static_cast<PFN_cuTensorMapEncodeTiled_v12000>(nullptr);
  }();
  return fn;
}

bool make_map(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer, uint64_t ld, uint32_t box_inner,
              uint32_t box_outer) {
  PFN_cuTensorMapEncodeTiled_v12000 enc = encode_fn();
  if (!enc) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {ld * 2};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  const CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                         CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool make_map_f32(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer, uint64_t ld, uint32_t box_inner,
                  uint32_t box_outer) {
  PFN_cuTensorMapEncodeTiled_v12000 enc = encode_fn();
  if (!enc) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {ld * 4};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  const CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<void*>(base), dims, strides, box, estr,
                         CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}
}  // namespace tc

namespace {

constexpr int BM = 128, BK = 64;
using namespace tc;

// --------------------------------------------------------------- epilogue
__device__ __forceinline__ void swiglu_bwd_chunk(const GemmArgs& a, int row, int j, const float (&dh)[32]);
__device__ __forceinline__ void relu2_chunk(const GemmArgs& a, int row, int j, const float (&v)[32]);

__device__ __forceinline__ void store_chunk(const GemmArgs& a, int row, int col, const float (&v)[32]) {
  if (a.epi == EPI_SWIGLU_BWD) {
    swiglu_bwd_chunk(a, row, col, v);
  } else if (a.epi == EPI_RELU2 || a.epi == EPI_RELU2_BWD) {
    relu2_chunk(a, row, col, v);
  } else if (a.epi == EPI_STORE_F32) {
    float4* p = reinterpret_cast<float4*>(static_cast<float*>(a.D) + (size_t)row * a.ldd + col);
#pragma unroll
    for (int i = 0; i < 8; ++i)
      p[i] = make_float4(a.alpha * v[4 * i], a.alpha * v[4 * i + 1], a.alpha * v[4 * i + 2], a.alpha * v[4 * i + 3]);
  } else if (a.epi == EPI_STORE || a.epi == EPI_ROPE) {
    uint4* p = reinterpret_cast<uint4*>(static_cast<bf16*>(a.D) + (size_t)row * a.ldd + col);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      uint4 q;
      __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&q);
#pragma unroll
      for (int j = 0; j < 4; ++j) h[j] = __floats2bfloat162_rn(a.alpha * v[8 * i + 2 * j], a.alpha * v[8 * i + 2 * j + 1]);
      p[i] = q;
    }
  } else {  // EPI_RESID: x[r] += alpha * acc on the kept row r (float32); compact float32 copy
    const long long r = src_row(a.kept_idx, a.S, row);
    float4* ps = a.save ? reinterpret_cast<float4*>(static_cast<float*>(a.save) + (size_t)row * a.ld_save + col)
                        : nullptr;
    if (r < 0) {  // padding row of a per-token kept list: no residual row; zero copy
      if (ps)
        for (int i = 0; i < 8; ++i) ps[i] = make_float4(0.f, 0.f, 0.f, 0.f);
      return;
    }
    float4* px = reinterpret_cast<float4*>(a.x + r * a.ldx + col);
    const float4* pl = a.resid_src ? reinterpret_cast<const float4*>(a.resid_src + (size_t)row * a.ld_src + col) : px;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      float4 o = pl[i];
      o.x += a.alpha * v[4 * i + 0];
      o.y += a.alpha * v[4 * i + 1];
      o.z += a.alpha * v[4 * i + 2];
      o.w += a.alpha * v[4 * i + 3];
      if (!a.x_skip) px[i] = o;
      if (ps) ps[i] = o;
    }
  }
}

__device__ __forceinline__ float silu_mul(float g, float u) { return g / (1.0f + expf(-g)) * u; }

__device__ __forceinline__ void st_bf16x32(bf16* dst, const float* v) {
  uint4* p = reinterpret_cast<uint4*>(dst);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    uint4 q;
    __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&q);
#pragma unroll
    for (int j = 0; j < 4; ++j) h[j] = __floats2bfloat162_rn(v[8 * i + 2 * j], v[8 * i + 2 * j + 1]);
    p[i] = q;
  }
}
__device__ __forceinline__ void ld_bf16x32(const bf16* src, float* v) {
  const uint4* p = reinterpret_cast<const uint4*>(src);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const uint4 q = p[i];
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&q);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float2 f = __bfloat1622float2(h[j]);
      v[8 * i + 2 * j] = f.x;
      v[8 * i + 2 * j + 1] = f.y;
    }
  }
}

// SwiGLU backward on a 32-column chunk of dh (hidden units j .. j+31).
__device__ __forceinline__ void swiglu_bwd_chunk(const GemmArgs& a, int row, int j, const float (&dh)[32]) {
  const bf16* gp = static_cast<const bf16*>(a.gu) + (size_t)row * 2 * a.F + j;
  float g[32], u[32], dg[32], du[32];
  ld_bf16x32(gp, g);
  ld_bf16x32(gp + a.F, u);
#pragma unroll
  for (int e = 0; e < 32; ++e) {
    const float sg = 1.0f / (1.0f + expf(-g[e]));
    dg[e] = dh[e] * u[e] * sg * (1.0f + g[e] * (1.0f - sg));
    du[e] = dh[e] * g[e] * sg;
  }
  bf16* dp = static_cast<bf16*>(a.D) + (size_t)row * 2 * a.F + j;
  st_bf16x32(dp, dg);
  st_bf16x32(dp + a.F, du);
}

// Squared ReLU on a 32-column chunk: forward (u -> save u, h = max(u,0)^2)
// or backward (dh -> du = dh * 2 max(u, 0) with the saved u).
__device__ __forceinline__ void relu2_chunk(const GemmArgs& a, int row, int j, const float (&v)[32]) {
  const size_t off = (size_t)row * a.ldd + j;
  float w[32];
  if (a.epi == EPI_RELU2) {
    float u[32];
#pragma unroll
    for (int e = 0; e < 32; ++e) {
      u[e] = v[e];
      const float r = fmaxf(v[e], 0.f);
      w[e] = r * r;
    }
    st_bf16x32(static_cast<bf16*>(a.D) + off, u);
    st_bf16x32(static_cast<bf16*>(a.h_out) + off, w);
  } else {
    float u[32];
    ld_bf16x32(static_cast<const bf16*>(a.gu) + off, u);
#pragma unroll
    for (int e = 0; e < 32; ++e) w[e] = v[e] * 2.f * fmaxf(u[e], 0.f);
    st_bf16x32(static_cast<bf16*>(a.D) + off, w);
  }
}

// Tile order: groups of 8 N-blocks; inside a group consecutive tiles walk
// the group's N-blocks for one M-block, then the next M-block, so the CTAs
// running at the same time share both A and B tiles in L2.
__device__ __forceinline__ void tile_coords(int tile, int num_m, int num_n, int& mb, int& nb) {
  constexpr int G = 8;
  const int grp = tile / (G * num_m);
  const int first_n = grp * G;
  const int gn = min(num_n - first_n, G);
  const int r = tile - grp * G * num_m;
  mb = r / gn;
  nb = first_n + r % gn;
}

// PAIR = false: one CTA per BM x BN tile, tcgen05.mma.cta_group::1.
// PAIR = true: a cluster of two CTAs (the two SMs of a TPC) shares a tile of
// 2*BM x BN.  Each CTA loads its own BM rows of A and half of the BN rows of
// B, so per k-step a CTA streams 32 KB instead of 48 KB from L2 and a stage
// takes 32 KB of shared memory (a deeper ring fits); the even CTA issues
// tcgen05.mma.cta_group::2 (M = 256) for both, and each CTA's TMEM receives
// its own BM rows of the accumulator, which its epilogue warps store.
// A ring stage holds KPS consecutive 64-deep k-blocks (each laid out as A
// then B); the MMA thread takes one barrier hand-off per stage, so KPS = 2
// halves the hand-offs per MMA (the tensor pipe queues only a few MMAs, and
// each hand-off costs a few hundred cycles of barrier latency).
template <int BN, int STAGES, bool A_MN, bool B_MN, bool PAIR, int KPS>
__global__ void __launch_bounds__(192, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const GemmArgs a) {
  constexpr int NCTA = PAIR ? 2 : 1;
  constexpr int BN_L = BN / NCTA;  // rows of B this CTA loads
  constexpr int BMT = BM * NCTA;   // rows of a tile
  constexpr uint32_t A_BYTES = BM * BK * 2;
  constexpr uint32_t B_BYTES = BN_L * BK * 2;
  constexpr uint32_t SUB_BYTES = A_BYTES + B_BYTES;  // one 64-deep k-block
  constexpr uint32_t STAGE_BYTES = KPS * SUB_BYTES;
  constexpr uint32_t TMEM_COLS = 2 * BN;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
  uint64_t* empty = full + STAGES;
  uint64_t* tfull = empty + STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = PAIR ? (cluster_rank() & 1u) : 0u;
  const int tile0 = PAIR ? (int)(blockIdx.x >> 1) : (int)blockIdx.x;
  const int tstep = PAIR ? (int)(gridDim.x >> 1) : (int)gridDim.x;
  const int M = a.M_cnt ? (*a.M_cnt) * a.M_mul : a.M;
  const int K = a.K_cnt ? (*a.K_cnt) * a.K_mul : a.K;
  const int N = a.N;
  const int num_m = (M + BMT - 1) / BMT, num_n = (N + BN - 1) / BN;
  const int num_tiles = num_m * num_n;
  const int num_kb = K / BK;                     // 64-deep k-blocks
  const int num_ks = (num_kb + KPS - 1) / KPS;  // ring stages per tile

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&tfull[s], 1);
      mbar_init(&tempty[s], 4 * NCTA);  // one lane of every epilogue warp of the tile's CTAs
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    if constexpr (PAIR)
      tmem_alloc_pair(tmem_slot, TMEM_COLS);
    else
      tmem_alloc(tmem_slot, TMEM_COLS);
  }
  tc_fence_before();
  __syncthreads();
  if constexpr (PAIR) cluster_sync();  // the peer's barriers are initialised before any remote arrival
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (num_kb == 0) {
    // Empty contraction (a layer that kept no sequence): the product is 0.
    if (warp >= 2) {
      const int q = warp & 3;
      float z[32];
#pragma unroll
      for (int i = 0; i < 32; ++i) z[i] = 0.f;
      for (int tile = tile0; tile < num_tiles; tile += tstep) {
        int mb, nb;
        tile_coords(tile, num_m, num_n, mb, nb);
        const int row = mb * BMT + (int)rank * BM + q * 32 + lane;
        for (int c = 0; c < BN; c += 32)
          if (row < M && nb * BN + c < N) store_chunk(a, row, nb * BN + c, z);
      }
    }
  } else if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------ TMA producer
      int stage = 0;
      uint32_t phase = 0;
      long long issued = 0;
      bool ok = true;
      for (int tile = tile0; tile < num_tiles && ok; tile += tstep) {
        int mb, nb;
        tile_coords(tile, num_m, num_n, mb, nb);
        const int arow = mb * BMT + (int)rank * BM;
        const int brow = nb * BN + (int)rank * BN_L;
        for (int ks = 0; ks < num_ks; ++ks) {
          if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, a.status)) {
            ok = false;
            break;
          }
          const int nk = min(KPS, num_kb - ks * KPS);  // k-blocks in this stage
          if constexpr (PAIR) {
            // both CTAs' copies complete on the even CTA's full barrier,
            // which the even CTA's MMA thread waits on
            if (rank == 0) mbar_arrive_expect_tx(&full[stage], 2u * (uint32_t)nk * SUB_BYTES);
          } else {
            mbar_arrive_expect_tx(&full[stage], (uint32_t)nk * SUB_BYTES);
          }
          for (int j = 0; j < nk; ++j) {
            const int kb = ks * KPS + j;
            uint8_t* sa = smem + stage * STAGE_BYTES + j * SUB_BYTES;
            uint8_t* sb = sa + A_BYTES;
            if constexpr (PAIR) {
              const uint32_t fb = cluster_addr(&full[stage], 0);
              if (!A_MN) {
                tma_load_2d_pair(sa, &tmA, kb * BK, arow, fb);
              } else {
                tma_load_2d_pair(sa, &tmA, arow, kb * BK, fb);
                tma_load_2d_pair(sa + 8192, &tmA, arow + 64, kb * BK, fb);
              }
              if (!B_MN && a.epi == EPI_SWIGLU) {
                // gate rows in the even CTA, the matching up rows in the odd one
                tma_load_2d_pair(sb, &tmB, kb * BK, (rank ? a.F : 0) + nb * BN_L, fb);
              } else if (!B_MN) {
                tma_load_2d_pair(sb, &tmB, kb * BK, brow, fb);
              } else {
#pragma unroll
                for (int c = 0; c < BN_L / 64; ++c) tma_load_2d_pair(sb + c * 8192, &tmB, brow + c * 64, kb * BK, fb);
              }
            } else {
              if (!A_MN) {
                tma_load_2d(sa, &tmA, kb * BK, arow, &full[stage]);
              } else {
                tma_load_2d(sa, &tmA, arow, kb * BK, &full[stage]);
                tma_load_2d(sa + 8192, &tmA, arow + 64, kb * BK, &full[stage]);
              }
              if (!B_MN && a.epi == EPI_SWIGLU) {
                // gate rows and up rows of the same hidden units side by side
                tma_load_2d(sb, &tmB, kb * BK, nb * (BN / 2), &full[stage]);
                tma_load_2d(sb + (BN / 2) * 128, &tmB, kb * BK, a.F + nb * (BN / 2), &full[stage]);
              } else if (!B_MN) {
                tma_load_2d(sb, &tmB, kb * BK, brow, &full[stage]);
              } else {
#pragma unroll
                for (int c = 0; c < BN / 64; ++c) tma_load_2d(sb + c * 8192, &tmB, brow + c * 64, kb * BK, &full[stage]);
              }
            }
          }
          ++issued;
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      const long long first = issued > STAGES ? issued - STAGES : 0;
      if (!ok && rank == 0) {
        // wait (bounded) for the copies still in flight (a pair's copies all
        // complete on the even CTA's barriers)
        for (long long i = first; i < issued; ++i) mbar_drain(&full[i % STAGES], (uint32_t)((i / STAGES) & 1));
      }
      if constexpr (PAIR) {
        // the even CTA's MMA commits arrive on these barriers of both CTAs:
        // wait (bounded) until the last ones have landed before the CTA ends
        for (long long i = first; i < issued; ++i) mbar_drain(&empty[i % STAGES], (uint32_t)((i / STAGES) & 1));
      }
    }
  } else if (warp == 1) {
    if (rank == 0) {
      // ------------------------------------------------ MMA issuer (whole warp, converged;
      // one elected lane issues)
      constexpr uint32_t IDESC = idesc_bf16(BMT, BN, A_MN, B_MN);
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool ok = true;
      for (int tile = tile0; tile < num_tiles && ok; tile += tstep) {
        if (!mbar_wait_conv<PAIR>(&tempty[acc], acc_phase ^ 1u, abort_flag, a.status)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * BN);
        for (int ks = 0; ks < num_ks; ++ks) {
          if (!mbar_wait_conv(&full[stage], phase, abort_flag, a.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const int nk = min(KPS, num_kb - ks * KPS);
#pragma unroll
          for (int j = 0; j < KPS; ++j) {
            if (j >= nk) break;
            const uint32_t sa = smem_u32(smem + stage * STAGE_BYTES + j * SUB_BYTES);
            const uint32_t sb = sa + A_BYTES;
#pragma unroll
            for (int k = 0; k < BK / 16; ++k) {
              // K-major: +32 bytes per 16-element K step inside the 128-byte
              // swizzle row.  MN-major: +16 rows of 128 bytes; 64-element MN
              // chunks 8 KB apart (LBO), 8-row groups 1 KB apart (SBO).
              const uint64_t ad = A_MN ? sdesc(sa + k * 2048, 8192, 1024) : sdesc(sa + k * 32, 16, 1024);
              const uint64_t bd = B_MN ? sdesc(sb + k * 2048, 8192, 1024) : sdesc(sb + k * 32, 16, 1024);
              const uint32_t accum = (ks | j | k) != 0 ? 1u : 0u;
              if constexpr (PAIR)
                mma_bf16_pair_w(d_tmem, ad, bd, IDESC, accum);
              else
                mma_bf16_w(d_tmem, ad, bd, IDESC, accum);
            }
          }
          if constexpr (PAIR)
            mma_commit_pair_both_w(&empty[stage]);
          else
            mma_commit_w(&empty[stage]);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        if constexpr (PAIR)
          mma_commit_pair_both_w(&tfull[acc]);
        else
          mma_commit_w(&tfull[acc]);
        acc ^= 1;
        if (acc == 0) acc_phase ^= 1u;
      }
      if (!ok) {
        // make sure every MMA issued so far has finished before TMEM is freed
        if constexpr (PAIR)
          mma_commit_pair_local_w(drain);
        else
          mma_commit_w(drain);
        if (lane == 0) mbar_drain(drain, 0);
        __syncwarp();
      }
    }
  } else {
    // ------------------------------------------------ epilogue (warps 2..5)
    const int q = warp & 3;  // TMEM lane quadrant this warp may access
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int tile = tile0; tile < num_tiles; tile += tstep) {
      int mb, nb;
      tile_coords(tile, num_m, num_n, mb, nb);
      // one lane waits; the warp follows its verdict (tcgen05.ld below is
      // warp-collective, so the whole warp must take the same path)
      int ok = 1;
      if (lane == 0) ok = mbar_wait(&tfull[acc], acc_phase, abort_flag, a.status) ? 1 : 0;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) break;
      tc_fence_after();
      const int row = mb * BMT + (int)rank * BM + q * 32 + lane;
      const uint32_t tbase = tmem_base + (uint32_t)(acc * BN) + ((uint32_t)(q * 32) << 16);
      if (a.epi == EPI_SWIGLU) {
        // columns [0, BN/2) hold g, [BN/2, BN) hold u of hidden units j0 + c
        const int j0 = nb * (BN / 2);
#pragma unroll 1
        for (int c = 0; c < BN / 2; c += 32) {
          float g[32], u[32], hv[32];
          tmem_ld32(tbase + (uint32_t)c, g);
          tmem_ld32(tbase + (uint32_t)(BN / 2 + c), u);
          if (row < M) {
#pragma unroll
            for (int e = 0; e < 32; ++e) hv[e] = silu_mul(g[e], u[e]);
            bf16* gp = static_cast<bf16*>(a.D) + (size_t)row * 2 * a.F + j0 + c;
            st_bf16x32(gp, g);
            st_bf16x32(gp + a.F, u);
            st_bf16x32(static_cast<bf16*>(a.h_out) + (size_t)row * a.F + j0 + c, hv);
          }
        }
      } else if (a.epi == EPI_ROPE) {
        // rotate pairs (i, i + Dh/2) of every q / k head in the tile
        const int half = a.Dh / 2;
        const int pos = row_pos(a.pos_tok, a.S, row);
#pragma unroll 1
        for (int hb = 0; hb < BN; hb += a.Dh) {
          const int col = nb * BN + hb;
#pragma unroll 1
          for (int c0 = 0; c0 < half; c0 += 32) {
            float x1[32], x2[32];
            tmem_ld32(tbase + (uint32_t)(hb + c0), x1);
            tmem_ld32(tbase + (uint32_t)(hb + half + c0), x2);
            if (row < M && col < N) {
              if (col < a.rope_cols) {
                const float4* cp = reinterpret_cast<const float4*>(a.rope_cos + (size_t)pos * half + c0);
                const float4* sp = reinterpret_cast<const float4*>(a.rope_sin + (size_t)pos * half + c0);
#pragma unroll
                for (int q4 = 0; q4 < 8; ++q4) {
                  const float4 cv = cp[q4], sv = sp[q4];
                  const float cs[4] = {cv.x, cv.y, cv.z, cv.w}, sn[4] = {sv.x, sv.y, sv.z, sv.w};
#pragma unroll
                  for (int k = 0; k < 4; ++k) {
                    const int e = 4 * q4 + k;
                    const float p1 = x1[e], p2 = x2[e];
                    x1[e] = p1 * cs[k] - p2 * sn[k];
                    x2[e] = p2 * cs[k] + p1 * sn[k];
                  }
                }
              }
              bf16* dp = static_cast<bf16*>(a.D) + (size_t)row * a.ldd + col;
              st_bf16x32(dp + c0, x1);
              st_bf16x32(dp + half + c0, x2);
            }
          }
        }
      } else if (a.epi == EPI_RESID) {
        // residual rows are read ahead (the next chunk while this one is
        // finished) so their latency overlaps the TMEM loads and the adds
        const long long rs = row < M ? src_row(a.kept_idx, a.S, row) : 0;
        const bool pad = row < M && rs < 0;  // padding row of a per-token kept list: zero copy only
        const bool rok = row < M && !pad;
        const long long r = rok ? rs : 0;
        // the old value comes from x[r], or from the compact copy resid_src
        float* xrow = a.x_skip ? nullptr : a.x + r * a.ldx + (size_t)nb * BN;
        const float* lrow = a.resid_src ? a.resid_src + (size_t)(row < M ? row : 0) * a.ld_src + (size_t)nb * BN
                                        : a.x + r * a.ldx + (size_t)nb * BN;
        float* srow = a.save ? static_cast<float*>(a.save) + (size_t)row * a.ld_save + (size_t)nb * BN : nullptr;
        float4 xv[8];
        if (rok && nb * BN < N) {
#pragma unroll
          for (int i = 0; i < 8; ++i) xv[i] = reinterpret_cast<const float4*>(lrow)[i];
        }
#pragma unroll 1
        for (int c = 0; c < BN; c += 32) {
          float v[32];
          tmem_ld32(tbase + (uint32_t)c, v);
          const bool ok = rok && nb * BN + c < N;
          float4 o[8];
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            o[i] = xv[i];
            o[i].x += a.alpha * v[4 * i + 0];
            o[i].y += a.alpha * v[4 * i + 1];
            o[i].z += a.alpha * v[4 * i + 2];
            o[i].w += a.alpha * v[4 * i + 3];
          }
          if (rok && c + 32 < BN && nb * BN + c + 32 < N) {
#pragma unroll
            for (int i = 0; i < 8; ++i) xv[i] = reinterpret_cast<const float4*>(lrow + c + 32)[i];
          }
          if (ok) {
            if (xrow) {
#pragma unroll
              for (int i = 0; i < 8; ++i) reinterpret_cast<float4*>(xrow + c)[i] = o[i];
            }
            if (srow) {
#pragma unroll
              for (int i = 0; i < 8; ++i) reinterpret_cast<float4*>(srow + c)[i] = o[i];
            }
          } else if (pad && srow && nb * BN + c < N) {
#pragma unroll
            for (int i = 0; i < 8; ++i) reinterpret_cast<float4*>(srow + c)[i] = make_float4(0.f, 0.f, 0.f, 0.f);
          }
        }
      } else if (a.epi == EPI_SWIGLU_BWD) {
        // the saved g and u of the next chunk are read while this one is
        // finished (as the residual epilogue does), so their latency overlaps
        // the TMEM load and the arithmetic
        const bool rowok = row < M;
        const bf16* gp = static_cast<const bf16*>(a.gu) + (size_t)(rowok ? row : 0) * 2 * a.F + (size_t)nb * BN;
        uint4 gq[4], uq[4];
        if (rowok && nb * BN < N) {
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            gq[i] = reinterpret_cast<const uint4*>(gp)[i];
            uq[i] = reinterpret_cast<const uint4*>(gp + a.F)[i];
          }
        }
#pragma unroll 1
        for (int c = 0; c < BN; c += 32) {
          float dh[32];
          tmem_ld32(tbase + (uint32_t)c, dh);
          const bool ok = rowok && nb * BN + c < N;
          float g[32], u[32];
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const __nv_bfloat162* g2 = reinterpret_cast<const __nv_bfloat162*>(&gq[i]);
            const __nv_bfloat162* u2 = reinterpret_cast<const __nv_bfloat162*>(&uq[i]);
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              const float2 gf = __bfloat1622float2(g2[k]), uf = __bfloat1622float2(u2[k]);
              g[8 * i + 2 * k] = gf.x;
              g[8 * i + 2 * k + 1] = gf.y;
              u[8 * i + 2 * k] = uf.x;
              u[8 * i + 2 * k + 1] = uf.y;
            }
          }
          if (rowok && c + 32 < BN && nb * BN + c + 32 < N) {
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              gq[i] = reinterpret_cast<const uint4*>(gp + c + 32)[i];
              uq[i] = reinterpret_cast<const uint4*>(gp + a.F + c + 32)[i];
            }
          }
          if (ok) {
            float du[32];  // dg is written over dh
#pragma unroll
            for (int e = 0; e < 32; ++e) {
              const float sg = 1.0f / (1.0f + expf(-g[e]));
              du[e] = dh[e] * g[e] * sg;
              dh[e] = dh[e] * u[e] * sg * (1.0f + g[e] * (1.0f - sg));
            }
            bf16* dp = static_cast<bf16*>(a.D) + (size_t)row * 2 * a.F + nb * BN + c;
            st_bf16x32(dp, dh);
            st_bf16x32(dp + a.F, du);
          }
        }
      } else {
#pragma unroll 1
        for (int c = 0; c < BN; c += 32) {
          float v[32];
          tmem_ld32(tbase + (uint32_t)c, v);
          if (row < M && nb * BN + c < N) store_chunk(a, row, nb * BN + c, v);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if constexpr (PAIR)
          mbar_arrive_cluster(cluster_addr(&tempty[acc], 0));
        else
          mbar_arrive(&tempty[acc]);
      }
      acc ^= 1;
      if (acc == 0) acc_phase ^= 1u;
    }
  }

  tc_fence_before();
  __syncthreads();
  if constexpr (PAIR) {
    // neither CTA ends (and frees its TMEM and shared memory) while the
    // other may still address them
    __syncwarp();
    cluster_sync();
  }
  if (warp == 1) {
    tc_fence_after();
    if constexpr (PAIR)
      tmem_dealloc_pair(tmem_base, TMEM_COLS);
    else
      tmem_dealloc(tmem_base, TMEM_COLS);
  }
}

template <int BN, int STAGES, bool PAIR, int KPS>
constexpr size_t smem_bytes() {
  return (size_t)STAGES * KPS * (BM * BK * 2 + (BN / (PAIR ? 2 : 1)) * BK * 2) + 1024 + 256;
}

// Tensor cores of the pair kernels: co-resident clusters of two CTAs (0 if
// the pair kernel cannot run).
constexpr int PAIR_BN = 256, PAIR_STAGES = 3, PAIR_KPS = 2;
int pair_clusters() {
  // once per process (initialisation of a function-local static is thread-safe)
  static const int clusters = [] {
    int n = 0;
    auto k = gemm_tc_kernel<PAIR_BN, PAIR_STAGES, false, false, true, PAIR_KPS>;
    constexpr size_t smem = smem_bytes<PAIR_BN, PAIR_STAGES, true, PAIR_KPS>();
    if (cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) == cudaSuccess) {
      cudaLaunchConfig_t cfg = {};
      cudaLaunchAttribute at[1];
      at[0].id = cudaLaunchAttributeClusterDimension;
      at[0].val.clusterDim.x = 2;
      at[0].val.clusterDim.y = 1;
      at[0].val.clusterDim.z = 1;
      cfg.gridDim = dim3(2);
      cfg.blockDim = dim3(192);
      cfg.dynamicSmemBytes = smem;
      cfg.attrs = at;
      cfg.numAttrs = 1;
      int c = 0;
      if (cudaOccupancyMaxActiveClusters(&c, k, &cfg) == cudaSuccess && c > 0) n = c;
    }
    cudaGetLastError();  // a refused query leaves no sticky error behind
    return n;
  }();
  return clusters;
}

template <int BN, int STAGES, bool A_MN, bool B_MN, bool PAIR, int KPS>
cudaError_t run(const GemmArgs& a, const CUtensorMap& ta, const CUtensorMap& tb, cudaStream_t st) {
  constexpr size_t smem = smem_bytes<BN, STAGES, PAIR, KPS>();
  constexpr int NCTA = PAIR ? 2 : 1;
  auto kern = gemm_tc_kernel<BN, STAGES, A_MN, B_MN, PAIR, KPS>;
  // once per process (initialisation of a function-local static is thread-safe)
  static const cudaError_t attr =
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (attr != cudaSuccess) return attr;
  const int mcap = a.M_cnt ? a.M_cap : a.M;
  const long long tiles = (long long)((mcap + BM * NCTA - 1) / (BM * NCTA)) * ((a.N + BN - 1) / BN);
  int units = PAIR ? pair_clusters() : device_sm_count();
  if (tiles < units) units = (int)(tiles > 0 ? tiles : 1);
  if constexpr (!PAIR) {
    kern<<<units, 192, smem, st>>>(ta, tb, a);
  } else {
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = 2;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.gridDim = dim3(2 * units);
    cfg.blockDim = dim3(192);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    cudaError_t e = cudaLaunchKernelEx(&cfg, kern, ta, tb, a);
    if (e != cudaSuccess) return e;
  }
  return cudaGetLastError();
}

template <int BN, int STAGES, bool PAIR, int KPS>
cudaError_t dispatch_major(const GemmArgs& a, const CUtensorMap& ta, const CUtensorMap& tb, cudaStream_t st) {
  if (!a.a_mn && !a.b_mn) return run<BN, STAGES, false, false, PAIR, KPS>(a, ta, tb, st);
  if (!a.a_mn && a.b_mn) return run<BN, STAGES, false, true, PAIR, KPS>(a, ta, tb, st);
  if (a.a_mn && !a.b_mn) return run<BN, STAGES, true, false, PAIR, KPS>(a, ta, tb, st);
  return run<BN, STAGES, true, true, PAIR, KPS>(a, ta, tb, st);
}

}  // namespace

// One block waiting on an mbarrier phase that nothing completes: the
// bounded wait gives up after its limit and records LD_ERR_TIMEOUT.
__global__ void wait_timeout_kernel(int* status) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    tc::mbar_init(&bar, 1);
    abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  if (threadIdx.x == 0) tc::mbar_wait(&bar, 0, reinterpret_cast<volatile int*>(&abort_flag), status);
}

cudaError_t launch_wait_timeout(int* status, cudaStream_t st) {
  wait_timeout_kernel<<<1, 32, 0, st>>>(status);
  return cudaGetLastError();
}

cudaError_t gemm_tc(const GemmArgs& a, cudaStream_t st) {
  const int BN = (a.N % 256 == 0) ? 256 : 128;
  const uint64_t mcap = a.M_cnt ? a.M_cap : a.M;
  const uint64_t kcap = a.K_cnt ? a.K_cap : a.K;
  if (mcap == 0 || a.N == 0) return cudaSuccess;
  // 256-column tiles run on CTA pairs where the device can co-schedule them
  const bool pair = BN == PAIR_BN && pair_clusters() > 0;
  CUtensorMap ta, tb;
  bool ok;
  // A(m,k): K-major = rows m of k; MN-major = rows k of m.
  if (!a.a_mn)
    ok = make_map(&ta, a.A, kcap ? kcap : 64, mcap, a.lda, 64, 128);
  else
    ok = make_map(&ta, a.A, mcap, kcap ? kcap : 64, a.lda, 64, 64);
  if (!ok) return cudaErrorInvalidValue;
  if (!a.b_mn)
    ok = make_map(&tb, a.B, kcap ? kcap : 64, a.N, a.ldb, 64,
                  (uint32_t)((a.epi == EPI_SWIGLU || pair) ? BN / 2 : BN));
  else
    ok = make_map(&tb, a.B, a.N, kcap ? kcap : 64, a.ldb, 64, 64);
  if (!ok) return cudaErrorInvalidValue;
  if (pair) return dispatch_major<PAIR_BN, PAIR_STAGES, true, PAIR_KPS>(a, ta, tb, st);
  if (BN == 256) return dispatch_major<256, 4, false, 1>(a, ta, tb, st);
  return dispatch_major<128, 3, false, 2>(a, ta, tb, st);
}

}  // namespace ldk
