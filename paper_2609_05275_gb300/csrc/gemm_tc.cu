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
//               B (BN x 64) into a STAGES-deep shared-memory ring;
//   warp 1      allocates 2*BN TMEM columns (two accumulators) and issues
//               tcgen05.mma (M=128, N=BN, K=16) from one thread;
//   warps 2..5  epilogue: tcgen05.ld of the accumulator (each warp reads
//               its 32-lane quadrant), fused scale / residual update, and
//               global stores, overlapped with the next tile's MMAs.
// Operands may be K-major or MN-major (weight-gradient and data-gradient
// products read activations and weights transposed); the shared-memory
// descriptors and the instruction descriptor's major bits cover both, so no
// transpose is ever materialised.
//
// Every mbarrier wait is bounded: after kWaitLimitNs the CTA raises the
// status word (LD_ERR_TIMEOUT), drains its own TMA copies and MMAs with a
// further bounded wait, frees its TMEM and exits.
#include <cuda.h>
#include <cudaTypedefs.h>

#include "ld_internal.cuh"

namespace ldk {
namespace {

constexpr int BM = 128, BK = 64;
constexpr uint32_t kDrainLimitNs = 200000000ull;

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// ---------------------------------------------------------------- mbarrier
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t addr, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.b32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(addr), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

// Bounded wait for the phase of parity `parity`.  False if the time limit
// passed (the block's abort flag and the status word are raised) or another
// role of the block aborted first.
__device__ __noinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag, int* status) {
  const uint32_t addr = smem_u32(bar);
  if (mbar_try_wait(addr, parity)) return true;
  const uint64_t t0 = gtimer_ns();
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait(addr, parity)) return true;
    if ((it & 31) == 0) {
      if (*abort_flag) return false;
      if (gtimer_ns() - t0 > kWaitLimitNs) {
        *abort_flag = 1;
        set_status(status, LD_ERR_TIMEOUT);
        return false;
      }
    }
  }
}
// Bounded wait used while draining after an abort (ignores the flag).
__device__ __noinline__ void mbar_drain(uint64_t* bar, uint32_t parity) {
  const uint32_t addr = smem_u32(bar);
  const uint64_t t0 = gtimer_ns();
  while (!mbar_try_wait(addr, parity)) {
    if (gtimer_ns() - t0 > kDrainLimitNs) return;
  }
}

// --------------------------------------------------------------------- TMA
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* tm, int c0, int c1, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
          smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(tm)), "r"(c0), "r"(c1), "r"(smem_u32(bar))
      : "memory");
}

// ----------------------------------------------------------------- tcgen05
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// Shared-memory matrix descriptor, 128-byte swizzle (layout type 2),
// descriptor version 1 (bits 46-47), base offset 0 (tiles are 1024-aligned).
__device__ __forceinline__ uint64_t sdesc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)((lbo >> 4) & 0x3FFFu) << 16) |
         ((uint64_t)((sbo >> 4) & 0x3FFFu) << 32) | (1ull << 46) | (2ull << 61);
}

// Instruction descriptor of kind::f16: fp32 accumulator (bits 4-5 = 1),
// A and B bf16 (bits 7-9 = 1, 10-12 = 1), A/B major (bits 15/16: 1 =
// MN-major), N >> 3 at bits 17-22, M >> 4 at bits 24-28.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N, bool a_mn, bool b_mn) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((a_mn ? 1u : 0u) << 15) | ((b_mn ? 1u : 0u) << 16) |
         ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                         uint32_t accum) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(
          d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accum)
      : "memory");
}
__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
               : "memory");
}

// 32 lanes x 32 consecutive fp32 columns of TMEM -> 32 registers per thread.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%"
      "19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
        "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr)
      : "memory");
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// --------------------------------------------------------------- epilogue
__device__ __forceinline__ void store_chunk(const GemmArgs& a, int row, int col, const float (&v)[32]) {
  if (a.epi == EPI_STORE_F32) {
    float4* p = reinterpret_cast<float4*>(static_cast<float*>(a.D) + (size_t)row * a.ldd + col);
#pragma unroll
    for (int i = 0; i < 8; ++i)
      p[i] = make_float4(a.alpha * v[4 * i], a.alpha * v[4 * i + 1], a.alpha * v[4 * i + 2], a.alpha * v[4 * i + 3]);
  } else if (a.epi == EPI_STORE) {
    uint4* p = reinterpret_cast<uint4*>(static_cast<bf16*>(a.D) + (size_t)row * a.ldd + col);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      uint4 q;
      __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&q);
#pragma unroll
      for (int j = 0; j < 4; ++j) h[j] = __floats2bfloat162_rn(a.alpha * v[8 * i + 2 * j], a.alpha * v[8 * i + 2 * j + 1]);
      p[i] = q;
    }
  } else {  // EPI_RESID: x[r] += alpha * acc on the kept row r; save the result
    const long long r = src_row(a.kept_idx, a.S, row);
    uint4* px = reinterpret_cast<uint4*>(static_cast<bf16*>(a.x) + r * a.ldx + col);
    uint4* ps = a.save ? reinterpret_cast<uint4*>(static_cast<bf16*>(a.save) + (size_t)row * a.ld_save + col)
                       : nullptr;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      uint4 q = px[i];
      __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&q);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const float2 old = __bfloat1622float2(h[j]);
        h[j] = __floats2bfloat162_rn(old.x + a.alpha * v[8 * i + 2 * j], old.y + a.alpha * v[8 * i + 2 * j + 1]);
      }
      px[i] = q;
      if (ps) ps[i] = q;
    }
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

template <int BN, int STAGES, bool A_MN, bool B_MN>
__global__ void __launch_bounds__(192, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const GemmArgs a) {
  constexpr uint32_t A_BYTES = BM * BK * 2;
  constexpr uint32_t B_BYTES = BN * BK * 2;
  constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
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
  const int M = a.M_cnt ? (*a.M_cnt) * a.M_mul : a.M;
  const int K = a.K_cnt ? (*a.K_cnt) * a.K_mul : a.K;
  const int N = a.N;
  const int num_m = (M + BM - 1) / BM, num_n = (N + BN - 1) / BN;
  const int num_tiles = num_m * num_n;
  const int num_kb = K / BK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&tfull[s], 1);
      mbar_init(&tempty[s], 4);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (num_kb == 0) {
    // Empty contraction (a layer that kept no sequence): the product is 0.
    if (warp >= 2) {
      const int q = warp & 3;
      float z[32];
#pragma unroll
      for (int i = 0; i < 32; ++i) z[i] = 0.f;
      for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x) {
        int mb, nb;
        tile_coords(tile, num_m, num_n, mb, nb);
        const int row = mb * BM + q * 32 + lane;
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
      for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x) {
        int mb, nb;
        tile_coords(tile, num_m, num_n, mb, nb);
        for (int kb = 0; kb < num_kb; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, a.status)) {
            ok = false;
            break;
          }
          uint8_t* sa = smem + stage * STAGE_BYTES;
          uint8_t* sb = sa + A_BYTES;
          mbar_arrive_expect_tx(&full[stage], STAGE_BYTES);
          if (!A_MN) {
            tma_load_2d(sa, &tmA, kb * BK, mb * BM, &full[stage]);
          } else {
            tma_load_2d(sa, &tmA, mb * BM, kb * BK, &full[stage]);
            tma_load_2d(sa + 8192, &tmA, mb * BM + 64, kb * BK, &full[stage]);
          }
          if (!B_MN) {
            tma_load_2d(sb, &tmB, kb * BK, nb * BN, &full[stage]);
          } else {
#pragma unroll
            for (int c = 0; c < BN / 64; ++c) tma_load_2d(sb + c * 8192, &tmB, nb * BN + c * 64, kb * BK, &full[stage]);
          }
          ++issued;
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (!ok) {
        // wait (bounded) for the copies this thread still has in flight
        for (long long i = issued > STAGES ? issued - STAGES : 0; i < issued; ++i)
          mbar_drain(&full[i % STAGES], (uint32_t)((i / STAGES) & 1));
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ------------------------------------------------ MMA issuer
      constexpr uint32_t IDESC = idesc_bf16(BM, BN, A_MN, B_MN);
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x) {
        if (!mbar_wait(&tempty[acc], acc_phase ^ 1u, abort_flag, a.status)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * BN);
        for (int kb = 0; kb < num_kb; ++kb) {
          if (!mbar_wait(&full[stage], phase, abort_flag, a.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + stage * STAGE_BYTES);
          const uint32_t sb = sa + A_BYTES;
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            // K-major: +32 bytes per 16-element K step inside the 128-byte
            // swizzle row.  MN-major: +16 rows of 128 bytes; 64-element MN
            // chunks 8 KB apart (LBO), 8-row groups 1 KB apart (SBO).
            const uint64_t ad = A_MN ? sdesc(sa + k * 2048, 8192, 1024) : sdesc(sa + k * 32, 16, 1024);
            const uint64_t bd = B_MN ? sdesc(sb + k * 2048, 8192, 1024) : sdesc(sb + k * 32, 16, 1024);
            mma_bf16(d_tmem, ad, bd, IDESC, (kb | k) != 0 ? 1u : 0u);
          }
          mma_commit(&empty[stage]);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        mma_commit(&tfull[acc]);
        acc ^= 1;
        if (acc == 0) acc_phase ^= 1u;
      }
      if (!ok) {
        // make sure every MMA issued so far has finished before TMEM is freed
        mma_commit(drain);
        mbar_drain(drain, 0);
      }
    }
  } else {
    // ------------------------------------------------ epilogue (warps 2..5)
    const int q = warp & 3;  // TMEM lane quadrant this warp may access
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x) {
      int mb, nb;
      tile_coords(tile, num_m, num_n, mb, nb);
      // one lane waits; the warp follows its verdict (tcgen05.ld below is
      // warp-collective, so the whole warp must take the same path)
      int ok = 1;
      if (lane == 0) ok = mbar_wait(&tfull[acc], acc_phase, abort_flag, a.status) ? 1 : 0;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) break;
      tc_fence_after();
      const int row = mb * BM + q * 32 + lane;
      const uint32_t tbase = tmem_base + (uint32_t)(acc * BN) + ((uint32_t)(q * 32) << 16);
#pragma unroll 1
      for (int c = 0; c < BN; c += 32) {
        float v[32];
        tmem_ld32(tbase + (uint32_t)c, v);
        if (row < M && nb * BN + c < N) store_chunk(a, row, nb * BN + c, v);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[acc]);
      acc ^= 1;
      if (acc == 0) acc_phase ^= 1u;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(TMEM_COLS) : "memory");
  }
}

// ---------------------------------------------------------------- host side
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// 2-D bf16 tensor map: `inner` contiguous elements per line, `outer` lines
// `ld` elements apart, box of box_inner x box_outer, 128-byte swizzle.
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

template <int BN, int STAGES, bool A_MN, bool B_MN>
cudaError_t run(const GemmArgs& a, const CUtensorMap& ta, const CUtensorMap& tb, cudaStream_t st) {
  constexpr size_t smem = (size_t)STAGES * (BM * BK * 2 + BN * BK * 2) + 1024 + 256;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(gemm_tc_kernel<BN, STAGES, A_MN, B_MN>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  const int mcap = a.M_cnt ? a.M_cap : a.M;
  const long long tiles = (long long)((mcap + BM - 1) / BM) * ((a.N + BN - 1) / BN);
  int grid = device_sm_count();
  if (tiles < grid) grid = (int)(tiles > 0 ? tiles : 1);
  gemm_tc_kernel<BN, STAGES, A_MN, B_MN><<<grid, 192, smem, st>>>(ta, tb, a);
  return cudaGetLastError();
}

template <int BN, int STAGES>
cudaError_t dispatch_major(const GemmArgs& a, const CUtensorMap& ta, const CUtensorMap& tb, cudaStream_t st) {
  if (!a.a_mn && !a.b_mn) return run<BN, STAGES, false, false>(a, ta, tb, st);
  if (!a.a_mn && a.b_mn) return run<BN, STAGES, false, true>(a, ta, tb, st);
  if (a.a_mn && !a.b_mn) return run<BN, STAGES, true, false>(a, ta, tb, st);
  return run<BN, STAGES, true, true>(a, ta, tb, st);
}

}  // namespace

cudaError_t gemm_tc(const GemmArgs& a, cudaStream_t st) {
  const int BN = (a.N % 256 == 0) ? 256 : 128;
  const uint64_t mcap = a.M_cnt ? a.M_cap : a.M;
  const uint64_t kcap = a.K_cnt ? a.K_cap : a.K;
  if (mcap == 0 || a.N == 0) return cudaSuccess;
  CUtensorMap ta, tb;
  bool ok;
  // A(m,k): K-major = rows m of k; MN-major = rows k of m.
  if (!a.a_mn)
    ok = make_map(&ta, a.A, kcap ? kcap : 64, mcap, a.lda, 64, 128);
  else
    ok = make_map(&ta, a.A, mcap, kcap ? kcap : 64, a.lda, 64, 64);
  if (!ok) return cudaErrorInvalidValue;
  if (!a.b_mn)
    ok = make_map(&tb, a.B, kcap ? kcap : 64, a.N, a.ldb, 64, (uint32_t)BN);
  else
    ok = make_map(&tb, a.B, a.N, kcap ? kcap : 64, a.ldb, 64, 64);
  if (!ok) return cudaErrorInvalidValue;
  if (BN == 256) return dispatch_major<256, 4>(a, ta, tb, st);
  return dispatch_major<128, 6>(a, ta, tb, st);
}

}  // namespace ldk
