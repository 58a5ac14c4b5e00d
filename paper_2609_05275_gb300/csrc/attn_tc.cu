// Causal grouped-query flash attention, forward, on the tcgen05 tensor cores
// (sm_103a), head sizes 64 and 128, sequence lengths that are multiples of
// 128.
//
// f_attn of Eq. (transformer_layer_dropout_train) for one kept sequence and
// query head h (key/value head g = floor(h*Hkv/H)):
//   o_i = sum_{j<=i} softmax_j(c q_i . k_j) v_j,  c = 1/sqrt(Dh);
// lse_i = log sum_j exp(c q_i . k_j) is kept for the backward.
//
// One CTA per (128-query tile, head, kept sequence); 320 threads:
//   warp 0      TMA: the Q tile once, then K_j and V_j tiles (128 keys) into
//               a three-stage K ring and a two-stage V ring (128-byte
//               swizzled, 64-column slabs), K one tile ahead of V;
//   warp 1      TMEM allocation and the MMAs: S_j = Q K_j^T into one of two
//               TMEM score buffers, then O += P_{j-1} V_{j-1} (O in TMEM,
//               P read from TMEM as the A operand);
//   warps 2..9  softmax, one query row and 64 keys per thread (two warps
//               per row): S_j from TMEM, running max in base 2,
//               P = exp2(S c log2e - m) written as bf16 into one of two TMEM
//               P buffers, so step j is written while P_{j-1} V_{j-1} runs.
// TMEM columns: S 0-255 (two buffers), O 256-(256+DH), P 384-511 (two).
// The running max is only moved (and O rescaled in TMEM) when it grows by
// more than 2^8, so most tiles need no O round trip; P <= 2^8 stays well
// inside bf16/fp32 range.  All waits are bounded (status word on expiry).
// With ALiBi (the paper's architecture, Methodology section) head h adds
// m_h (j - i) to the scaled score of query i and key j: the scores are first
// turned into biased base-2 logits x = S c log2e + m_h log2e (j - i), and the
// max and P = exp2(x - m) work on x.
// The two warps of a row pass their partial maxima through tagged 64-bit
// shared-memory words (tile index, value), a bounded spin per tile.
// With per-token kept lists a sequence is a segment of arbitrary length
// (seg[b] .. seg[b+1]-1); rows of a tile past its end are never stored.
#include <type_traits>

#include "tc_common.cuh"

namespace ldk {
namespace {
using namespace tc;

constexpr uint32_t SLAB = 128 * 128;  // bytes of a 128-row x 64-column bf16 slab
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr float kRescale = 8.0f;  // move the running max only when it grows by > 2^8

__device__ __forceinline__ void st_volatile_u64(uint64_t* p, uint64_t v) {
  asm volatile("st.volatile.shared.u64 [%0], %1;" ::"r"(smem_u32(p)), "l"(v) : "memory");
}
__device__ __forceinline__ uint64_t ld_volatile_u64(const uint64_t* p) {
  uint64_t v;
  asm volatile("ld.volatile.shared.u64 %0, [%1];" : "=l"(v) : "r"(smem_u32(p)) : "memory");
  return v;
}
// Warp-uniform bounded wait for a (tag << 32 | value) word written by a
// partner thread: true with the value once every lane's word carries `tag`;
// false (abort flag and status raised) after kWaitLimitNs or when another
// role aborted.
__device__ __forceinline__ bool xchg_wait(const uint64_t* p, uint32_t tag, float& v, volatile int* abort_flag,
                                          int* status) {
  uint64_t w = ld_volatile_u64(p);
  if (__all_sync(0xffffffffu, (uint32_t)(w >> 32) == tag)) {
    v = __uint_as_float((uint32_t)w);
    return true;
  }
  const uint64_t t0 = gtimer_ns();
  for (uint32_t it = 1;; ++it) {
    w = ld_volatile_u64(p);
    if (__all_sync(0xffffffffu, (uint32_t)(w >> 32) == tag)) {
      v = __uint_as_float((uint32_t)w);
      return true;
    }
    if ((it & 255) == 0) {
      int bad = 0;
      if ((threadIdx.x & 31) == 0) {
        bad = *abort_flag ? 1 : 0;
        if (!bad && gtimer_ns() - t0 > kWaitLimitNs) {
          *abort_flag = 1;
          set_status(status, LD_ERR_TIMEOUT);
          bad = 1;
        }
      }
      if (__shfl_sync(0xffffffffu, bad, 0)) return false;
    }
  }
}

__device__ __forceinline__ void st_bf16x32_(bf16* dst, const float* v) {
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
// byte offset of element (row r, 16-byte chunk i) in a 128B-swizzled
// K-major slab of 128-byte rows
__device__ __forceinline__ uint32_t swz(int r, int i) {
  return (uint32_t)((r >> 3) * 1024 + (r & 7) * 128 + (((i & 7) ^ (r & 7)) << 4));
}

template <int DH, bool ALIBI>
__global__ void __launch_bounds__(320, 1)
    attn_fwd_tc_kernel(const __grid_constant__ CUtensorMap tm, bf16* __restrict__ o, int ldo, float* __restrict__ lse,
                       int lse_ld, const int* __restrict__ cnt, int S, int H, int Hkv,
                       const float* __restrict__ alibi, const int* __restrict__ seg, int* status) {
  constexpr int NSLAB = DH / 64;
  constexpr uint32_t TILE = NSLAB * SLAB;  // one 128 x DH bf16 tile
  constexpr int NSK = 3, NSV = 2;          // K and V stages
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* Qs = smem;
  uint8_t* Ks = Qs + TILE;
  uint8_t* Vs = Ks + NSK * TILE;
  uint8_t* xch = Vs + NSV * TILE;
  // row-max exchange words (tile index << 32 | max bits), [tile parity][half][row]
  uint64_t(*xmax)[2][128] = reinterpret_cast<uint64_t(*)[2][128]>(xch);
  float(*xsum)[128] = reinterpret_cast<float(*)[128]>(xch + 2 * 2 * 128 * 8);  // [half][row]
  uint64_t* bars = reinterpret_cast<uint64_t*>(xch + 10 * 128 * 4);
  uint64_t* q_full = bars;
  uint64_t* k_full = bars + 1;        // [NSK] K ring: a stage frees once S_j has read it
  uint64_t* k_empty = k_full + NSK;
  uint64_t* v_full = k_empty + NSK;   // [NSV] V ring: a stage frees once P_j V_j has read it
  uint64_t* v_empty = v_full + NSV;
  uint64_t* s_full = v_empty + NSV;
  uint64_t* s_free = s_full + 2;
  uint64_t* p_full = s_free + 2;      // [2] per P buffer
  uint64_t* pv_done = p_full + 2;     // [2] per P buffer
  uint64_t* o_full = pv_done + 2;
  uint64_t* drain = o_full + 1;
  uint64_t* xbar = drain + 1;  // [4]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(xbar + 4);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  // sequence: rows row0 .. row0+len-1 (a whole kept sequence, or with `seg`
  // the kept tokens of sequence blockIdx.y); the rows of the last tile past
  // len belong to other sequences: causality hides them from the valid
  // queries, and their own results are not stored
  const int seq = blockIdx.y;
  int row0, len;
  if (seg) {
    row0 = seg[seq];
    len = seg[seq + 1] - row0;
  } else {
    if (seq >= *cnt) return;
    row0 = seq * S;
    len = S;
  }
  const int nqt = S / 128;
  const int qt = nqt - 1 - blockIdx.z;  // slowest grid dimension: heaviest tiles are dispatched first
  if (qt * 128 >= len) return;
  const int h = blockIdx.x, g = (h * Hkv) / H;
  const int nkt = qt + 1;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int s = 0; s < NSK; ++s) {
      mbar_init(&k_full[s], 1);
      mbar_init(&k_empty[s], 1);
    }
    for (int s = 0; s < NSV; ++s) {
      mbar_init(&v_full[s], 1);
      mbar_init(&v_empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&s_full[b], 1);
      mbar_init(&s_free[b], 8);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&p_full[b], 8);
      mbar_init(&pv_done[b], 1);
    }
    mbar_init(o_full, 1);
    mbar_init(drain, 1);
    for (int q = 0; q < 4; ++q) mbar_init(&xbar[q], 2);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  for (int i = threadIdx.x; i < 2 * 2 * 128; i += blockDim.x) (&xmax[0][0][0])[i] = ~0ull;  // no tile yet
  if (warp == 1) tmem_alloc(tmem_slot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t t_o = tmem + 256;  // O accumulator: columns 256 .. 256+DH
  const uint32_t t_p = tmem + 384;  // [2] x 64 columns: P as bf16 pairs (A operand of P V)

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------ TMA producer
      const int qcol = h * DH, kcol = (H + g) * DH, vcol = (H + Hkv + g) * DH;
      mbar_arrive_expect_tx(q_full, TILE);
      for (int c = 0; c < NSLAB; ++c) tma_load_2d(Qs + c * SLAB, &tm, qcol + 64 * c, row0 + qt * 128, q_full);
      // K runs one tile ahead of V: S_{j+1} is issued before P_j V_j
      int nk = 0, nv = 0;
      for (int j = 0; j <= nkt; ++j) {
        if (j < nkt) {
          const int s = j % NSK;
          if (!mbar_wait(&k_empty[s], ((j / NSK) & 1) ^ 1u, abort_flag, status)) break;
          mbar_arrive_expect_tx(&k_full[s], TILE);
          for (int c = 0; c < NSLAB; ++c)
            tma_load_2d(Ks + s * TILE + c * SLAB, &tm, kcol + 64 * c, row0 + j * 128, &k_full[s]);
          ++nk;
        }
        if (j >= 1) {
          const int jv = j - 1, s = jv % NSV;
          if (!mbar_wait(&v_empty[s], ((jv / NSV) & 1) ^ 1u, abort_flag, status)) break;
          mbar_arrive_expect_tx(&v_full[s], TILE);
          for (int c = 0; c < NSLAB; ++c)
            tma_load_2d(Vs + s * TILE + c * SLAB, &tm, vcol + 64 * c, row0 + jv * 128, &v_full[s]);
          ++nv;
        }
      }
      if (*abort_flag) {
        mbar_drain(q_full, 0);
        for (int j = nk > NSK ? nk - NSK : 0; j < nk; ++j) mbar_drain(&k_full[j % NSK], (j / NSK) & 1);
        for (int j = nv > NSV ? nv - NSV : 0; j < nv; ++j) mbar_drain(&v_full[j % NSV], (j / NSV) & 1);
      }
    }
  } else if (warp == 1) {
    {  // the whole warp, converged; one elected lane issues
      // ------------------------------------------------ MMA issuer
      constexpr uint32_t ID_S = idesc_bf16(128, 128, false, false);  // S = Q K^T
      constexpr uint32_t ID_O = idesc_bf16(128, DH, false, true);    // O += P V (V MN-major)
      // descriptors built once, advanced by (byte offset >> 4) per MMA
      const uint64_t DQ = sdesc(smem_u32(Qs), 16, 1024), DK = sdesc(smem_u32(Ks), 16, 1024);
      const uint64_t DV = sdesc(smem_u32(Vs), SLAB, 1024);
      bool ok = mbar_wait_conv(q_full, 0, abort_flag, status);
      for (int j = 0; ok && j <= nkt; ++j) {
        if (j < nkt) {
          const int s = j % NSK;
          if (!mbar_wait_conv(&k_full[s], (j / NSK) & 1, abort_flag, status)) { ok = false; break; }
          if (!mbar_wait_conv(&s_free[j & 1], ((j >> 1) & 1) ^ 1u, abort_flag, status)) { ok = false; break; }
          tc_fence_after();
          const uint64_t kb = DK + (uint64_t)((s * TILE) >> 4);
#pragma unroll
          for (int kk = 0; kk < DH / 16; ++kk) {
            const uint32_t off = ((kk >> 2) * SLAB + (kk & 3) * 32) >> 4;
            mma_bf16_w(tmem + (j & 1) * 128, DQ + off, kb + off, ID_S, kk > 0);
          }
          mma_commit_w(&s_full[j & 1]);
          mma_commit_w(&k_empty[s]);
        }
        if (j >= 1) {
          const int jp = j - 1, s = jp % NSV, pb = jp & 1;
          if (!mbar_wait_conv(&p_full[pb], (jp >> 1) & 1, abort_flag, status)) { ok = false; break; }
          if (!mbar_wait_conv(&v_full[s], (jp / NSV) & 1, abort_flag, status)) { ok = false; break; }
          tc_fence_after();
          const uint64_t vb = DV + (uint64_t)((s * TILE) >> 4);
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) {
            // A = P from TMEM (16 keys = 8 columns a step); B = V as MN-major
            // (dh contiguous): 64-dh chunks one slab apart, 8-key groups 1 KB
            mma_bf16_ta_w(t_o, t_p + pb * 64 + kk * 8, vb + ((kk * 2048) >> 4), ID_O, (jp > 0 || kk > 0) ? 1u : 0u);
          }
          mma_commit_w(&pv_done[pb]);
          mma_commit_w(&v_empty[s]);
        }
      }
      if (ok) {
        mma_commit_w(o_full);
      } else {
        mma_commit_w(drain);
        if (lane == 0) mbar_drain(drain, 0);
        __syncwarp();
      }
    }
  } else {
    // ------------------------------------------------ softmax (warps 2..9)
    // two warps per TMEM lane quadrant, one query row per thread: warps 2..5
    // take keys 0..63 of the tile (and O columns 0..DH/2), warps 6..9 keys
    // 64..127 (and the rest of O); the pair exchanges row maxima and sums
    // through shared memory
    const int quad = warp & 3;
    const int half = (warp - 2) >> 2;
    const int r = quad * 32 + lane;  // query row of this thread within the tile
    const uint32_t lane_off = (uint32_t)(quad * 32) << 16;
    uint64_t* xb = &xbar[quad];      // exchange barrier of the two warps of this quadrant (2 arrivals a phase)
    // logits are x = S * sl2 (+ ALiBi bias); after the ALiBi transform the
    // scores held are already x, so the scale applied later is 1
    const float sl2 = kLog2e * rsqrtf((float)DH);
    const float sl2e = ALIBI ? 1.f : sl2;
    const float slope2 = ALIBI ? alibi[h] * kLog2e : 0.f;
    constexpr int OC = DH / 64;      // 32-column chunks of O per half
    float m_used = -INFINITY, l = 0.f;
    bool ok = true;
    for (int j = 0; j < nkt; ++j) {
      if (!warp_wait(&s_full[j & 1], (j >> 1) & 1, abort_flag, status)) { ok = false; break; }
      tc_fence_after();
      uint32_t sr[2][32];
      tmem_ld32_nw(tmem + (j & 1) * 128 + half * 64 + lane_off, sr[0]);
      tmem_ld32_nw(tmem + (j & 1) * 128 + half * 64 + 32 + lane_off, sr[1]);
      tmem_wait_ld();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&s_free[j & 1]);
      // running max on the raw scores (the scale is positive); keys after
      // the query (diagonal tile only) are left out
      const bool diag = (j == qt);                       // the only tile with masked keys (block-uniform)
      const int lim = (diag ? r : 127) - half * 64;      // last visible local column
      if constexpr (ALIBI) {
        // x_e = S_e sl2 + slope2 (key_e - query) for the 64 keys of this half
        const float b0 = slope2 * (float)(j * 128 + half * 64 - (qt * 128 + r));
        const uint64_t sl2x2 = f2_pack(sl2, sl2), sx2 = f2_pack(slope2, slope2), b0x2 = f2_pack(b0, b0);
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          float x0, x1;
          f2_unpack(f2_fma(f2_pack(__uint_as_float(sr[e >> 4][(2 * e) & 31]), __uint_as_float(sr[e >> 4][(2 * e + 1) & 31])),
                           sl2x2, f2_fma(f2_pack((float)(2 * e), (float)(2 * e + 1)), sx2, b0x2)),
                    x0, x1);
          sr[e >> 4][(2 * e) & 31] = __float_as_uint(x0);
          sr[e >> 4][(2 * e + 1) & 31] = __float_as_uint(x1);
        }
      }
      float mraw = -INFINITY;
      if (diag) {
#pragma unroll
        for (int e = 0; e < 64; ++e) mraw = fmaxf(mraw, e <= lim ? __uint_as_float(sr[e >> 5][e & 31]) : -INFINITY);
      } else {
#pragma unroll
        for (int e = 0; e < 64; e += 2)
          mraw = fmax3(mraw, __uint_as_float(sr[e >> 5][e & 31]), __uint_as_float(sr[e >> 5][(e & 31) + 1]));
      }
      // partner's max of this row through a (tile, value) word: a shared-
      // memory round trip instead of an mbarrier phase (whose arrival takes
      // a few hundred cycles to be seen); parity double-buffered, so a word
      // is rewritten only after the partner has passed the next exchange
      st_volatile_u64(&xmax[j & 1][half][r], ((uint64_t)(uint32_t)j << 32) | __float_as_uint(mraw));
      float pmax;
      if (!xchg_wait(&xmax[j & 1][half ^ 1][r], (uint32_t)j, pmax, abort_flag, status)) { ok = false; break; }
      mraw = fmaxf(mraw, pmax);
      const float mt = mraw * sl2e;
      const bool rescale = mt > m_used + kRescale;
      const float m_new = rescale ? mt : m_used;
      // P = exp2(S c log2e - m) on pairs of keys (packed fp32 pipe); the
      // causal mask only on the diagonal tile
      uint32_t pk[32];
      uint64_t ls2 = f2_pack(0.f, 0.f);
      auto pass = [&](auto masked) {
        constexpr bool MASK = decltype(masked)::value;
        const uint64_t sl2x2 = f2_pack(sl2e, sl2e), nm2 = f2_pack(-m_new, -m_new);
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          float x0, x1;
          f2_unpack(f2_fma(f2_pack(__uint_as_float(sr[e >> 4][(2 * e) & 31]), __uint_as_float(sr[e >> 4][(2 * e + 1) & 31])),
                           sl2x2, nm2),
                    x0, x1);
          float p0 = ex2(x0), p1 = ex2(x1);
          if constexpr (MASK) {
            p0 = (2 * e <= lim) ? p0 : 0.f;
            p1 = (2 * e + 1 <= lim) ? p1 : 0.f;
          }
          ls2 = f2_add(ls2, f2_pack(p0, p1));
          pk[e] = bf16x2_bits(p0, p1);
        }
      };
      if (diag) pass(std::true_type{});
      else pass(std::false_type{});
      float ls_a, ls_b;
      f2_unpack(ls2, ls_a, ls_b);
      const float ls = ls_a + ls_b;
      // P_{j-2} V_{j-2} must be done with P buffer j & 1 before it is
      // rewritten; O is rescaled only once P_{j-1} V_{j-1} has accumulated
      const int pb = j & 1;
      if (j >= 2 && !warp_wait(&pv_done[pb], ((j >> 1) & 1) ^ 1u, abort_flag, status)) { ok = false; break; }
      const bool any_rescale = j >= 1 && __any_sync(0xffffffffu, rescale);
      if (any_rescale && !warp_wait(&pv_done[pb ^ 1], ((j - 1) >> 1) & 1, abort_flag, status)) { ok = false; break; }
      tc_fence_after();
      // tcgen05.ld/st are warp-wide: the warp rescales its half of O together
      // when any lane moved its max; lanes that did not multiply by 1
      if (any_rescale) {
        const float corr = rescale ? exp2f(m_used - m_new) : 1.f;
#pragma unroll 1
        for (int c = 0; c < OC; ++c) {
          float t[32];
          tmem_ld32(t_o + half * (DH / 2) + c * 32 + lane_off, t);
#pragma unroll
          for (int e = 0; e < 32; ++e) t[e] *= corr;
          tmem_st32(t_o + half * (DH / 2) + c * 32 + lane_off, t);
        }
      }
      if (rescale) {
        l *= exp2f(m_used - m_new);
        m_used = m_new;
      }
      l += ls;
      // this half's 64 keys of row r -> columns 32 half .. 32 half + 31 of P buffer pb
      tmem_st32u(t_p + pb * 64 + half * 32 + lane_off, pk);
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&p_full[pb]);
    }
    if (ok && warp_wait(o_full, 0, abort_flag, status)) {
      tc_fence_after();
      xsum[half][r] = l;
      __syncwarp();
      if (lane == 0) mbar_arrive(xb);
      const bool got = warp_wait(xb, 0, abort_flag, status);  // the barrier's only phase
      const float lt = l + (got ? xsum[half ^ 1][r] : 0.f);
      const float inv = 1.0f / lt;
      const bool valid = qt * 128 + r < len;
      bf16* orow = o + (long long)(row0 + qt * 128 + r) * ldo + (long long)h * DH + half * (DH / 2);
#pragma unroll 1
      for (int c = 0; c < OC; ++c) {
        float t[32];
        tmem_ld32(t_o + half * (DH / 2) + c * 32 + lane_off, t);
        uint4* dst = reinterpret_cast<uint4*>(orow + c * 32);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          uint4 q;
          __nv_bfloat162* hb = reinterpret_cast<__nv_bfloat162*>(&q);
#pragma unroll
          for (int k = 0; k < 4; ++k) hb[k] = __floats2bfloat162_rn(t[8 * i + 2 * k] * inv, t[8 * i + 2 * k + 1] * inv);
          if (valid) dst[i] = q;
        }
      }
      if (half == 0 && valid) lse[(size_t)h * lse_ld + row0 + qt * 128 + r] = (m_used + log2f(lt)) * kLn2;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

template <int DH, bool ALIBI>
cudaError_t fwd_tc(const bf16* qkv, int ldq, bf16* o, int ldo, float* lse, const int* cnt, int S, int H, int Hkv,
                   int max_seqs, const float* alibi, const int* seg, int* status, cudaStream_t st) {
  // Q, 3 K and 2 V tiles + the row max / sum exchange + alignment + barriers
  constexpr size_t smem = (size_t)(DH / 64) * SLAB * 6 + 10 * 128 * 4 + 1024 + 256;
  // once per process (initialisation of a function-local static is thread-safe)
  static const cudaError_t attr =
      cudaFuncSetAttribute(attn_fwd_tc_kernel<DH, ALIBI>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (attr != cudaSuccess) return attr;
  CUtensorMap tm;
  if (!make_map(&tm, qkv, (uint64_t)ldq, (uint64_t)max_seqs * S, (uint64_t)ldq, 64, 128)) return cudaErrorInvalidValue;
  dim3 grid(H, max_seqs, S / 128);
  attn_fwd_tc_kernel<DH, ALIBI><<<grid, 320, smem, st>>>(tm, o, ldo, lse, max_seqs * S, cnt, S, H, Hkv, alibi, seg,
                                                         status);
  return cudaGetLastError();
}


// ---------------------------------------------------------------------------
// Forward, head size 128 (with or without the ALiBi bias): two 128-query
// tiles per CTA ("ping-pong").  Each tile has its own softmax group of four warps with one
// query row and all 128 keys of a K tile per thread, so no two warps share a
// row; the MMA warp alternates between the groups, and one group's softmax
// runs while the tensor pipe works for the other:
//   warp 0      TMA: both Q tiles once, then K_j and V_j (three-stage K ring,
//               two-stage V ring), K one tile ahead of V;
//   warp 1      TMEM allocation and, per K tile j: P_A(j-1) V_{j-1}, S_A(j) =
//               Q_A K_j^T, P_B(j-1) V_{j-1}, S_B(j) = Q_B K_j^T;
//   warps 2..5  softmax of tile A (the block's first 128 queries), warps
//               6..9 of tile B.
// TMEM columns: S_A 0-127, S_B 128-255, O_A 256-383, O_B 384-511.  P_g is
// written as bf16 pairs over the first 64 columns of S_g once S_g has been
// read (the next S_g MMA is issued after the P_g V MMA that reads it).  MMAs
// run in issue order, so S_g(j) complete implies P_g(j-1) V_{j-1} complete:
// the group may rescale O_g as soon as S_g(j) is ready.  Tile B is skipped
// when the sequence ends before it.
constexpr int PP_NSK = 3, PP_NSV = 2;
// Pairs (of the 16 in each 32-key chunk) whose exponentials run on the FMA
// pipe (ex2_poly2) instead of MUFU: the 128 x 128 exponentials of a tile
// take as many cycles at 16 a clock as the tile's two MMAs.
constexpr int PP_POLY = 0;

// 2^x for two values on the FMA pipe: x = n + f with n = rint(x) and f in
// [-1/2, 1/2]; 2^f = 1 + f (C1 + f (C2 + f C3)), the cubic fitted to 2^f on
// that interval by minimising the largest relative error (1.0e-4 in float32,
// below the 2^-9 half-ulp of the bf16 P is stored in); 2^n is added into the
// exponent field.  x is clamped at -127, where the result is below 2^-126
// instead of 0.
__device__ __forceinline__ void ex2_poly2(float x0, float x1, float& y0, float& y1) {
  constexpr float C1 = 0.6932829022407532f, C2 = 0.24221037328243256f, C3 = 0.05500858277082443f;
  x0 = fmaxf(x0, -127.f);
  x1 = fmaxf(x1, -127.f);
  const float n0 = rintf(x0), n1 = rintf(x1);
  const uint64_t f = f2_sub(f2_pack(x0, x1), f2_pack(n0, n1));
  uint64_t p = f2_fma(f, f2_pack(C3, C3), f2_pack(C2, C2));
  p = f2_fma(p, f, f2_pack(C1, C1));
  p = f2_fma(p, f, f2_pack(1.f, 1.f));
  float p0, p1;
  f2_unpack(p, p0, p1);
  y0 = __int_as_float(__float_as_int(p0) + ((int)n0 << 23));
  y1 = __int_as_float(__float_as_int(p1) + ((int)n1 << 23));
}

template <bool ALIBI>
__global__ void __launch_bounds__(320, 1)
    attn_fwd_pp_kernel(const __grid_constant__ CUtensorMap tm, bf16* __restrict__ o, int ldo, float* __restrict__ lse,
                       int lse_ld, const int* __restrict__ cnt, int S, int H, int Hkv,
                       const float* __restrict__ alibi, const int* __restrict__ seg, int* status) {
  constexpr int DH = 128;
  constexpr uint32_t TILE = 2 * SLAB;  // one 128 x 128 bf16 tile (two 64-column slabs)
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* Qs = smem;                 // [2] query tiles
  uint8_t* Ks = Qs + 2 * TILE;        // [PP_NSK]
  uint8_t* Vs = Ks + PP_NSK * TILE;   // [PP_NSV]
  uint64_t* bars = reinterpret_cast<uint64_t*>(Vs + PP_NSV * TILE);
  uint64_t* q_full = bars;
  uint64_t* k_full = q_full + 1;      // [PP_NSK]
  uint64_t* k_empty = k_full + PP_NSK;
  uint64_t* v_full = k_empty + PP_NSK;  // [PP_NSV]
  uint64_t* v_empty = v_full + PP_NSV;
  uint64_t* s_full = v_empty + PP_NSV;  // [2] per query tile
  uint64_t* p_full = s_full + 2;        // [2]
  uint64_t* o_full = p_full + 2;        // [2]
  uint64_t* drain = o_full + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int seq = blockIdx.y;
  int row0, len;
  if (seg) {
    row0 = seg[seq];
    len = seg[seq + 1] - row0;
  } else {
    if (seq >= *cnt) return;
    row0 = seq * S;
    len = S;
  }
  const int nqb = (S + 255) / 256;
  const int qb = nqb - 1 - blockIdx.z;  // heaviest query blocks first
  if (qb * 256 >= len) return;
  const bool vB = qb * 256 + 128 < len;  // tile B holds queries of the sequence
  const int nkA = 2 * qb + 1, nkB = vB ? 2 * qb + 2 : 0;  // K tiles of tile A / B (through its diagonal)
  const int nkt = vB ? nkB : nkA;
  const int h = blockIdx.x, g = (h * Hkv) / H;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int s = 0; s < PP_NSK; ++s) {
      mbar_init(&k_full[s], 1);
      mbar_init(&k_empty[s], 1);
    }
    for (int s = 0; s < PP_NSV; ++s) {
      mbar_init(&v_full[s], 1);
      mbar_init(&v_empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&s_full[b], 1);
      mbar_init(&p_full[b], 4);
      mbar_init(&o_full[b], 1);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(tmem_slot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------ TMA producer
      const int qcol = h * DH, kcol = (H + g) * DH, vcol = (H + Hkv + g) * DH;
      const int nq = vB ? 2 : 1;
      mbar_arrive_expect_tx(q_full, nq * TILE);
      for (int t = 0; t < nq; ++t)
        for (int c = 0; c < 2; ++c)
          tma_load_2d(Qs + t * TILE + c * SLAB, &tm, qcol + 64 * c, row0 + qb * 256 + t * 128, q_full);
      int nkl = 0, nvl = 0;
      for (int j = 0; j <= nkt; ++j) {
        if (j < nkt) {
          const int s = j % PP_NSK;
          if (!mbar_wait(&k_empty[s], ((j / PP_NSK) & 1) ^ 1u, abort_flag, status)) break;
          mbar_arrive_expect_tx(&k_full[s], TILE);
          for (int c = 0; c < 2; ++c)
            tma_load_2d(Ks + s * TILE + c * SLAB, &tm, kcol + 64 * c, row0 + j * 128, &k_full[s]);
          ++nkl;
        }
        if (j >= 1) {
          const int jv = j - 1, s = jv % PP_NSV;
          if (!mbar_wait(&v_empty[s], ((jv / PP_NSV) & 1) ^ 1u, abort_flag, status)) break;
          mbar_arrive_expect_tx(&v_full[s], TILE);
          for (int c = 0; c < 2; ++c)
            tma_load_2d(Vs + s * TILE + c * SLAB, &tm, vcol + 64 * c, row0 + jv * 128, &v_full[s]);
          ++nvl;
        }
      }
      if (*abort_flag) {
        mbar_drain(q_full, 0);
        for (int j = nkl > PP_NSK ? nkl - PP_NSK : 0; j < nkl; ++j) mbar_drain(&k_full[j % PP_NSK], (j / PP_NSK) & 1);
        for (int j = nvl > PP_NSV ? nvl - PP_NSV : 0; j < nvl; ++j) mbar_drain(&v_full[j % PP_NSV], (j / PP_NSV) & 1);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer (whole warp, converged; one elected lane issues)
    constexpr uint32_t ID_S = idesc_bf16(128, 128, false, false);  // S = Q K^T
    constexpr uint32_t ID_O = idesc_bf16(128, DH, false, true);    // O += P V (V MN-major)
    const uint64_t DQ = sdesc(smem_u32(Qs), 16, 1024), DK = sdesc(smem_u32(Ks), 16, 1024);
    const uint64_t DV = sdesc(smem_u32(Vs), SLAB, 1024);
    __syncwarp();
    bool ok = mbar_wait_conv(q_full, 0, abort_flag, status);
    for (int j = 0; ok && j <= nkt; ++j) {
      if (j < nkt && !mbar_wait_conv(&k_full[j % PP_NSK], (j / PP_NSK) & 1, abort_flag, status)) { ok = false; break; }
      if (j >= 1 && !mbar_wait_conv(&v_full[(j - 1) % PP_NSV], ((j - 1) / PP_NSV) & 1, abort_flag, status)) {
        ok = false;
        break;
      }
      for (int gi = 0; gi < 2; ++gi) {
        const int nkg = gi ? nkB : nkA;
        if (j >= 1 && j - 1 < nkg) {
          // O_g += P_g(j-1) V_{j-1}: A = P from the S_g columns, B = V MN-major
          if (!mbar_wait_conv(&p_full[gi], (j - 1) & 1, abort_flag, status)) { ok = false; break; }
          tc_fence_after();
          const uint64_t vb = DV + (uint64_t)((((j - 1) % PP_NSV) * TILE) >> 4);
#pragma unroll
          for (int kk = 0; kk < 8; ++kk)
            mma_bf16_ta_w(tmem + 256 + gi * 128, tmem + gi * 128 + kk * 8, vb + ((kk * 2048) >> 4), ID_O,
                            (j > 1 || kk > 0) ? 1u : 0u);
          if (j == nkg) mma_commit_w(&o_full[gi]);  // the group's last P V
        }
        if (j < nkg) {
          // S_g(j) = Q_g K_j^T, over the P_g the MMAs above have read
          const uint64_t kb = DK + (uint64_t)(((j % PP_NSK) * TILE) >> 4);
          const uint64_t qd = DQ + (uint64_t)((gi * TILE) >> 4);
#pragma unroll
          for (int kk = 0; kk < DH / 16; ++kk) {
            const uint32_t off = ((kk >> 2) * SLAB + (kk & 3) * 32) >> 4;
            mma_bf16_w(tmem + gi * 128, qd + off, kb + off, ID_S, kk > 0 ? 1u : 0u);
          }
          mma_commit_w(&s_full[gi]);
        }
      }
      if (!ok) break;
      if (j < nkt) mma_commit_w(&k_empty[j % PP_NSK]);
      if (j >= 1) mma_commit_w(&v_empty[(j - 1) % PP_NSV]);
    }
    if (!ok) {
      mma_commit_w(drain);
      if (lane == 0) mbar_drain(drain, 0);
      __syncwarp();
    }
  } else {
    // ------------------------------------------------ softmax (warps 2..9)
    const int gi = (warp - 2) >> 2;  // 0: tile A, 1: tile B
    const int quad = warp & 3;
    const int r = quad * 32 + lane;  // query row within the tile
    const uint32_t lane_off = (uint32_t)(quad * 32) << 16;
    const uint32_t t_s = tmem + gi * 128, t_og = tmem + 256 + gi * 128;
    const int nkg = gi ? nkB : nkA;
    const int jdiag = 2 * qb + gi;  // the K tile on this query tile's diagonal
    const float sl2 = kLog2e * rsqrtf((float)DH);
    // ALiBi: the exponent is x = S sl2 + slope2 (key - query), and the
    // running max m is kept on x (the max of S alone, scaled, otherwise)
    const float slope2 = ALIBI ? alibi[h] * kLog2e : 0.f;
    const int qrow_t = qb * 256 + gi * 128 + r;  // this thread's query within the sequence
    float m_used = -INFINITY, l = 0.f;
    bool ok = true;
    for (int j = 0; j < nkg; ++j) {
      if (!warp_wait(&s_full[gi], j & 1, abort_flag, status)) { ok = false; break; }
      tc_fence_after();
      const bool diag = (j == jdiag);  // keys after the query are left out (block-uniform)
      // pass 1: row max of the raw scores (the scale is positive), or of x
      // with ALiBi
      float mraw = -INFINITY;
      const float b0 = slope2 * (float)(j * 128 - qrow_t);  // bias of key 0 of the tile
#pragma unroll 1
      for (int c2 = 0; c2 < 2; ++c2) {
        uint32_t sr[2][32];
        tmem_ld32_nw(t_s + c2 * 64 + lane_off, sr[0]);
        tmem_ld32_nw(t_s + c2 * 64 + 32 + lane_off, sr[1]);
        tmem_wait_ld();
        if constexpr (ALIBI) {
          const uint64_t sl2x2 = f2_pack(sl2, sl2), sx2 = f2_pack(slope2, slope2);
          const float bc = b0 + slope2 * (float)(c2 * 64);
          const uint64_t bx2 = f2_pack(bc, bc);
#pragma unroll
          for (int e = 0; e < 64; e += 2) {
            float x0, x1;
            f2_unpack(f2_fma(f2_pack(__uint_as_float(sr[e >> 5][e & 31]), __uint_as_float(sr[e >> 5][(e & 31) + 1])),
                             sl2x2, f2_fma(f2_pack((float)e, (float)(e + 1)), sx2, bx2)),
                      x0, x1);
            sr[e >> 5][e & 31] = __float_as_uint(x0);
            sr[e >> 5][(e & 31) + 1] = __float_as_uint(x1);
          }
        }
        if (diag) {
#pragma unroll
          for (int e = 0; e < 64; ++e)
            mraw = fmaxf(mraw, c2 * 64 + e <= r ? __uint_as_float(sr[e >> 5][e & 31]) : -INFINITY);
        } else {
#pragma unroll
          for (int e = 0; e < 64; e += 2)
            mraw = fmax3(mraw, __uint_as_float(sr[e >> 5][e & 31]), __uint_as_float(sr[e >> 5][(e & 31) + 1]));
        }
      }
      const float mt = ALIBI ? mraw : mraw * sl2;
      const bool rescale = mt > m_used + kRescale;
      const float m_new = rescale ? mt : m_used;
      // O_g is rescaled in TMEM when any lane of the warp moved its max
      // (P_g(j-1) V_{j-1} is complete: it was issued before S_g(j))
      if (j >= 1 && __any_sync(0xffffffffu, rescale)) {
        const float corr = rescale ? exp2f(m_used - m_new) : 1.f;
#pragma unroll 1
        for (int c = 0; c < DH / 32; ++c) {
          float t[32];
          tmem_ld32(t_og + c * 32 + lane_off, t);
#pragma unroll
          for (int e = 0; e < 32; ++e) t[e] *= corr;
          tmem_st32(t_og + c * 32 + lane_off, t);
        }
      }
      if (rescale) {
        l *= exp2f(m_used - m_new);
        m_used = m_new;
      }
      // pass 2: P = exp2(S c log2e - m) for 32 keys at a time, written as
      // bf16 pairs over S columns that have already been read
      const uint64_t sl2x2 = f2_pack(sl2, sl2), nm2 = f2_pack(-m_new, -m_new);
      const uint64_t sx2 = f2_pack(slope2, slope2);
      uint64_t ls2 = f2_pack(0.f, 0.f);
#pragma unroll 1
      for (int c = 0; c < 4; ++c) {
        uint32_t sr[32];
        tmem_ld32_nw(t_s + c * 32 + lane_off, sr);
        tmem_wait_ld();
        uint32_t pk[16];
        const float bm = b0 + slope2 * (float)(c * 32) - m_new;  // ALiBi: bias of key 32c minus the max
        const uint64_t bmx2 = f2_pack(bm, bm);
#pragma unroll
        for (int e = 0; e < 16; ++e) {
          float x0, x1;
          const uint64_t add = ALIBI ? f2_fma(f2_pack((float)(2 * e), (float)(2 * e + 1)), sx2, bmx2) : nm2;
          f2_unpack(f2_fma(f2_pack(__uint_as_float(sr[2 * e]), __uint_as_float(sr[2 * e + 1])), sl2x2, add), x0, x1);
          float p0, p1;
          if (e >= 16 - PP_POLY) {
            ex2_poly2(x0, x1, p0, p1);
          } else {
            p0 = ex2(x0);
            p1 = ex2(x1);
          }
          if (diag) {
            p0 = (c * 32 + 2 * e <= r) ? p0 : 0.f;
            p1 = (c * 32 + 2 * e + 1 <= r) ? p1 : 0.f;
          }
          ls2 = f2_add(ls2, f2_pack(p0, p1));
          pk[e] = bf16x2_bits(p0, p1);
        }
        tmem_st16(t_s + c * 16 + lane_off, pk);  // keys 32c .. 32c+31 -> packed columns 16c .. 16c+15
      }
      tmem_wait_st();
      float ls_a, ls_b;
      f2_unpack(ls2, ls_a, ls_b);
      l += ls_a + ls_b;
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&p_full[gi]);
    }
    const bool has_tile = gi == 0 || vB;
    if (ok && has_tile && warp_wait(&o_full[gi], 0, abort_flag, status)) {
      tc_fence_after();
      const float inv = 1.0f / l;
      const int qrow = qb * 256 + gi * 128 + r;
      const bool valid = qrow < len;
      bf16* orow = o + (long long)(row0 + qrow) * ldo + (long long)h * DH;
#pragma unroll 1
      for (int c = 0; c < DH / 32; ++c) {
        float t[32];
        tmem_ld32(t_og + c * 32 + lane_off, t);
#pragma unroll
        for (int e = 0; e < 32; ++e) t[e] *= inv;
        if (valid) st_bf16x32_(orow + c * 32, t);
      }
      if (valid) lse[(size_t)h * lse_ld + row0 + qrow] = (m_used + log2f(l)) * kLn2;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

template <bool ALIBI>
cudaError_t fwd_pp(const bf16* qkv, int ldq, bf16* o, int ldo, float* lse, const int* cnt, int S, int H, int Hkv,
                   int max_seqs, const float* alibi, const int* seg, int* status, cudaStream_t st) {
  // 2 Q, 3 K and 2 V tiles of 32 KB + alignment + barriers = 230,656 bytes (of 232,448)
  constexpr size_t smem = (size_t)(2 + PP_NSK + PP_NSV) * 2 * SLAB + 1024 + 256;
  // once per process (initialisation of a function-local static is thread-safe)
  static const cudaError_t attr =
      cudaFuncSetAttribute(attn_fwd_pp_kernel<ALIBI>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (attr != cudaSuccess) return attr;
  CUtensorMap tm;
  if (!make_map(&tm, qkv, (uint64_t)ldq, (uint64_t)max_seqs * S, (uint64_t)ldq, 64, 128)) return cudaErrorInvalidValue;
  dim3 grid(H, max_seqs, (S + 255) / 256);
  attn_fwd_pp_kernel<ALIBI><<<grid, 320, smem, st>>>(tm, o, ldo, lse, max_seqs * S, cnt, S, H, Hkv, alibi, seg, status);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Backward, head size 128.  One CTA per (128-key tile, kv head, kept
// sequence), looping over the query heads of the group and the 64-query
// tiles at or after the key tile.  448 threads:
//   warp 0      TMA: K, V once; Q_i, dO_i, lse_i, D_i per step (3 stages)
//   warp 1      MMAs, one step ahead: S^T_i = K Q_i^T, dP^T_i = V dO_i^T
//               (M = 128 keys, N = 64 queries); then for step i-1
//               dV += P^T dO (P^T read from TMEM), dK += dS^T Q (M = 128
//               keys, N = 128) and dQ^T = K^T dS^T (M = 128 head dims,
//               N = 64 queries)
//   warps 2..9  one key and 32 queries per thread: P^T = exp2(S^T c log2e - lse log2e)
//               as bf16 into TMEM, dS^T = P^T (dP^T - D) as bf16 into a
//               swizzled shared-memory tile; at the end dK (times c) and dV
//               from TMEM to dqkv
//   warps 10..13  dQ^T from TMEM, added into the float32 dQ buffer
// P^T and dS^T are double-buffered (step i uses buffer i & 1), so the
// softmax warps write step i while the MMAs of step i-1 still read theirs.
// TMEM columns: S^T 0-63, dP^T 64-127, dV 128-255, dK 256-383, dQ^T 384-447,
// P^T 448-479 / 480-511.
constexpr uint32_t HSLAB = 64 * 128;  // bytes of a 64-row x 64-column bf16 slab

// Values 4 e4 .. 4 e4 + 3 of p (shared memory), read by every lane of the
// warp at the same address.  Four 32-bit shared-space loads: a generic
// 128-bit read of such a broadcast cost about ten shared-memory wavefronts
// (1,300 a step of the backward), an ld.shared.v4 about five, a 32-bit
// ld.shared one.
__device__ __forceinline__ float lds_f32(uint32_t a) {
  float v;
  asm volatile("ld.shared.f32 %0, [%1];" : "=f"(v) : "r"(a) : "memory");
  return v;
}
__device__ __forceinline__ float4 ld4s(const float* p, int e4) {
  const uint32_t a = smem_u32(p + 4 * e4);
  return make_float4(lds_f32(a), lds_f32(a + 4), lds_f32(a + 8), lds_f32(a + 12));
}

template <bool ALIBI>
__global__ void __launch_bounds__(448, 1)
    attn_bwd_tc_kernel(const __grid_constant__ CUtensorMap tmkv, const __grid_constant__ CUtensorMap tmq,
                       const __grid_constant__ CUtensorMap tmo, const __grid_constant__ CUtensorMap tmdq,
                       const float* __restrict__ lse, const float* __restrict__ Dvec, int lse_ld,
                       float* __restrict__ dq_acc, bf16* __restrict__ dqkv, int ldq, const int* __restrict__ cnt,
                       int S, int H, int Hkv, const float* __restrict__ rcos, const float* __restrict__ rsin,
                       const float* __restrict__ alibi, const int* __restrict__ seg, const int* __restrict__ tok,
                       int* status) {
  constexpr int DH = 128;
  constexpr uint32_t KT = 2 * SLAB;    // 128 keys x 128 dims
  constexpr uint32_t QT = 2 * HSLAB;   // 64 queries x 128 dims
  constexpr int NST = 3;               // stages of the Q / dO / lse / D ring
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* Ks = smem;
  uint8_t* Vs = Ks + KT;
  uint8_t* Qs = Vs + KT;         // [NST][QT]
  uint8_t* dOs = Qs + NST * QT;  // [NST][QT]
  uint8_t* DSs = dOs + NST * QT; // [2] 128 keys x 64 queries, one slab of 128-byte rows each
  float* dqs = reinterpret_cast<float*>(DSs + 2 * SLAB);  // [64 queries][128 dims] float32 staging (1 KB aligned)
  // [NST][lse 68 | D 68]: the 64 values of a step start at float `voff` of
  // each half (a sequence's rows start anywhere with per-token kept lists,
  // and a bulk copy needs a 16-byte aligned source, so 68 are copied from
  // the aligned-down address)
  float* vecs = dqs + 64 * DH;
  constexpr int VS = 136;
  uint64_t* bars = reinterpret_cast<uint64_t*>(vecs + NST * VS);
  uint64_t* kv_full = bars;
  uint64_t* ld_full = bars + 1;          // [NST]
  uint64_t* ld_empty = ld_full + NST;    // [NST]
  uint64_t* sdp_full = ld_empty + NST;
  uint64_t* sdp_free = sdp_full + 1;
  uint64_t* p_ready = sdp_full + 2;  // [2] per P^T / dS^T buffer
  uint64_t* mm_done = sdp_full + 4;  // [2] per P^T / dS^T buffer
  uint64_t* dq_free = sdp_full + 6;
  uint64_t* acc_done = sdp_full + 7;
  uint64_t* drain = sdp_full + 8;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sdp_full + 9);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  // rows row0 .. row0+len-1 as in the forward; queries past len (the last
  // query tile) get P = dS = 0, keys past len are never stored
  const int seq = blockIdx.z;
  int row0, len;
  if (seg) {
    row0 = seg[seq];
    len = seg[seq + 1] - row0;
  } else {
    if (seq >= *cnt) return;
    row0 = seq * S;
    len = S;
  }
  const int kt = blockIdx.y, g = blockIdx.x, grp = H / Hkv;
  if (kt * 128 >= len) return;
  const int nq = (len + 63) / 64, q0 = 2 * kt;  // query tiles q0 .. nq-1 overlap or follow the keys
  const int n_it = grp * (nq - q0);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    mbar_init(kv_full, 1);
    for (int b = 0; b < NST; ++b) {
      mbar_init(&ld_full[b], 1);
      mbar_init(&ld_empty[b], 1);
    }
    mbar_init(sdp_full, 1);
    mbar_init(sdp_free, 8);
    for (int b = 0; b < 2; ++b) {
      mbar_init(&p_ready[b], 8);
      mbar_init(&mm_done[b], 1);
    }
    mbar_init(dq_free, 4);
    mbar_init(acc_done, 1);
    mbar_init(drain, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(tmem_slot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t t_s = tmem, t_dp = tmem + 64, t_dv = tmem + 128, t_dk = tmem + 256, t_dq = tmem + 384;
  const uint32_t t_p = tmem + 448;  // [2] x 32 columns: P^T as bf16 pairs

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------ TMA producer
      const int kcol = (H + g) * DH, vcol = (H + Hkv + g) * DH;
      mbar_arrive_expect_tx(kv_full, 2 * KT);
      for (int c = 0; c < 2; ++c) {
        tma_load_2d(Ks + c * SLAB, &tmkv, kcol + 64 * c, row0 + kt * 128, kv_full);
        tma_load_2d(Vs + c * SLAB, &tmkv, vcol + 64 * c, row0 + kt * 128, kv_full);
      }
      int issued = 0;
      for (int i = 0; i < n_it; ++i) {
        const int b = i % NST;
        const int h = g * grp + i / (nq - q0), qt = q0 + i % (nq - q0);
        if (!mbar_wait(&ld_empty[b], ((i / NST) & 1) ^ 1u, abort_flag, status)) break;
        mbar_arrive_expect_tx(&ld_full[b], 2 * QT + 2 * 272);
        for (int c = 0; c < 2; ++c) {
          tma_load_2d(Qs + b * QT + c * HSLAB, &tmq, h * DH + 64 * c, row0 + qt * 64, &ld_full[b]);
          tma_load_2d(dOs + b * QT + c * HSLAB, &tmo, h * DH + 64 * c, row0 + qt * 64, &ld_full[b]);
        }
        const size_t vo = ((size_t)h * lse_ld + row0 + qt * 64) & ~(size_t)3;  // lse_ld % 4 == 0
        bulk_load(vecs + b * VS, lse + vo, 272, &ld_full[b]);
        bulk_load(vecs + b * VS + 68, Dvec + vo, 272, &ld_full[b]);
        ++issued;
      }
      if (*abort_flag) {
        mbar_drain(kv_full, 0);
        for (int i = issued > NST ? issued - NST : 0; i < issued; ++i) mbar_drain(&ld_full[i % NST], (i / NST) & 1);
      }
    }
  } else if (warp == 1) {
    {  // the whole warp, converged; one elected lane issues
      // ------------------------------------------------ MMA issuer
      constexpr uint32_t ID_SP = idesc_bf16(128, 64, false, false);   // S^T, dP^T
      constexpr uint32_t ID_KV = idesc_bf16(128, DH, false, true);    // dV, dK (B = dO / Q, MN-major)
      constexpr uint32_t ID_Q = idesc_bf16(128, 64, true, true);      // dQ^T (A = K, B = dS^T, MN-major)
      // shared-memory descriptors built once; an MMA's operand is its base
      // plus (byte offset >> 4) in the address field (every tile lies below
      // 256 KB, so the 14-bit field never carries)
      const uint64_t DK = sdesc(smem_u32(Ks), 16, 1024), DV = sdesc(smem_u32(Vs), 16, 1024);
      const uint64_t DQ = sdesc(smem_u32(Qs), 16, 1024), DO = sdesc(smem_u32(dOs), 16, 1024);
      const uint64_t DQMN = sdesc(smem_u32(Qs), HSLAB, 1024), DOMN = sdesc(smem_u32(dOs), HSLAB, 1024);
      const uint64_t DKMN = sdesc(smem_u32(Ks), SLAB, 1024), DS = sdesc(smem_u32(DSs), 16, 1024);
      bool ok = mbar_wait_conv(kv_full, 0, abort_flag, status);
      for (int i = 0; ok && i <= n_it; ++i) {
        if (i < n_it) {
          const int b = i % NST;
          if (!mbar_wait_conv(&ld_full[b], (i / NST) & 1, abort_flag, status)) { ok = false; break; }
          if (!mbar_wait_conv(sdp_free, (i & 1) ^ 1u, abort_flag, status)) { ok = false; break; }
          tc_fence_after();
          const uint64_t st = (uint64_t)((b * QT) >> 4);
#pragma unroll
          for (int kk = 0; kk < DH / 16; ++kk) {
            const uint32_t koff = ((kk >> 2) * SLAB + (kk & 3) * 32) >> 4;
            const uint32_t qoff = ((kk >> 2) * HSLAB + (kk & 3) * 32) >> 4;
            mma_bf16_w(t_s, DK + koff, DQ + st + qoff, ID_SP, kk > 0);
            mma_bf16_w(t_dp, DV + koff, DO + st + qoff, ID_SP, kk > 0);
          }
          mma_commit_w(sdp_full);
        }
        if (i >= 1) {
          const int ip = i - 1, b = ip % NST, pb = ip & 1;
          if (!mbar_wait_conv(&p_ready[pb], (ip >> 1) & 1, abort_flag, status)) { ok = false; break; }
          if (!mbar_wait_conv(dq_free, (ip & 1) ^ 1u, abort_flag, status)) { ok = false; break; }
          tc_fence_after();
          const uint64_t st = (uint64_t)((b * QT) >> 4), ds = (uint64_t)((pb * SLAB) >> 4);
          const uint32_t first = ip > 0 ? 1u : 0u;
#pragma unroll
          for (int kk = 0; kk < 4; ++kk) {  // contraction over the 64 queries
            const uint32_t aoff = (kk * 32) >> 4;                // dS^T, K-major
            const uint32_t boff = (kk * 2048) >> 4;              // dO / Q as MN-major
            mma_bf16_ta_w(t_dv, t_p + pb * 32 + kk * 8, DOMN + st + boff, ID_KV, kk > 0 ? 1u : first);
            mma_bf16_w(t_dk, DS + ds + aoff, DQMN + st + boff, ID_KV, kk > 0 ? 1u : first);
          }
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) {  // contraction over the 128 keys
            mma_bf16_w(t_dq, DKMN + ((kk * 2048) >> 4), DS + ds + ((kk * 2048) >> 4), ID_Q, kk > 0);
          }
          mma_commit_w(&mm_done[pb]);
          mma_commit_w(&ld_empty[b]);
        }
      }
      if (ok) {
        mma_commit_w(acc_done);
      } else {
        mma_commit_w(drain);
        if (lane == 0) mbar_drain(drain, 0);
        __syncwarp();
      }
    }
  } else if (warp < 10) {
    // ------------------------------------------------ P / dS (warps 2..9)
    // two warps per TMEM lane quadrant: warps 2..5 take queries 0..31 of the
    // step, warps 6..9 queries 32..63, one key per thread
    const int quad = warp & 3;
    const int half = (warp - 2) >> 2;
    const int r = quad * 32 + lane;  // key within the tile
    const int key = kt * 128 + r;
    const uint32_t lane_off = (uint32_t)(quad * 32) << 16;
    const int voff = row0 & 3;  // first value of a step in its lse / D stage (see vecs)
    const float sl2 = kLog2e * rsqrtf((float)DH);
    bool ok = true;
    for (int i = 0; i < n_it; ++i) {
      const int b = i % NST;
      const int qt = q0 + i % (nq - q0);
      // ALiBi: logit bias slope2 (key - query) of this step's query head
      const float slope2 = ALIBI ? alibi[g * grp + i / (nq - q0)] * kLog2e : 0.f;
      if (!warp_wait(sdp_full, i & 1, abort_flag, status)) { ok = false; break; }
      if (!warp_wait(&ld_full[b], (i / NST) & 1, abort_flag, status)) { ok = false; break; }
      tc_fence_after();
      uint32_t sr[32], dr[32];
      tmem_ld32_nw(t_s + half * 32 + lane_off, sr);
      tmem_ld32_nw(t_dp + half * 32 + lane_off, dr);
      tmem_wait_ld();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(sdp_free);
      const float* lsrc = vecs + b * VS + voff + half * 32;       // lse of the 32 queries
      const float* dsrc = vecs + b * VS + 68 + voff + half * 32;  // D of the 32 queries
      const int qbase = qt * 64 + half * 32 - key;  // query c is visible iff qbase + c >= 0
      const int qlim = len - (qt * 64 + half * 32);  // and exists iff c < qlim (warp-uniform)
      uint32_t pk[16], dk[16];
      // pairs of queries on the packed fp32 pipe; the mask only on warps
      // whose 32 keys are not all visible to the 32 queries, or whose queries
      // run past the sequence (warp-uniform)
      auto pass = [&](auto masked) {
        constexpr bool MASK = decltype(masked)::value;
        const uint64_t sl2x2 = f2_pack(sl2, sl2), nlog2 = f2_pack(-kLog2e, -kLog2e);
        // bias of query c: slope2 (key - qt*64 - half*32 - c) = b0 - slope2 c
        const float b0 = slope2 * (float)(-qbase);
        const uint64_t nsx2 = f2_pack(-slope2, -slope2), b0x2 = f2_pack(b0, b0);
#pragma unroll
        for (int e4 = 0; e4 < 8; ++e4) {
          const float4 lq = ld4s(lsrc, e4), dq = ld4s(dsrc, e4);
          uint64_t nl[2] = {f2_mul(f2_pack(lq.x, lq.y), nlog2), f2_mul(f2_pack(lq.z, lq.w), nlog2)};
          if constexpr (ALIBI) {
#pragma unroll
            for (int h2 = 0; h2 < 2; ++h2) {
              const float c0 = (float)(4 * e4 + 2 * h2);
              nl[h2] = f2_add(nl[h2], f2_fma(f2_pack(c0, c0 + 1.f), nsx2, b0x2));
            }
          }
          const uint64_t dd[2] = {f2_pack(dq.x, dq.y), f2_pack(dq.z, dq.w)};
#pragma unroll
          for (int h2 = 0; h2 < 2; ++h2) {
            const int c = 4 * e4 + 2 * h2;
            float x0, x1;
            f2_unpack(f2_fma(f2_pack(__uint_as_float(sr[c]), __uint_as_float(sr[c + 1])), sl2x2, nl[h2]), x0, x1);
            float p0 = ex2(x0), p1 = ex2(x1);
            const bool v0 = !MASK || (qbase + c >= 0 && c < qlim), v1 = !MASK || (qbase + c + 1 >= 0 && c + 1 < qlim);
            if constexpr (MASK) {
              p0 = v0 ? p0 : 0.f;
              p1 = v1 ? p1 : 0.f;
            }
            const uint64_t pp = f2_pack(p0, p1);
            float d0, d1;
            f2_unpack(f2_mul(pp, f2_sub(f2_pack(__uint_as_float(dr[c]), __uint_as_float(dr[c + 1])), dd[h2])), d0, d1);
            if constexpr (MASK) {  // rows past the sequence may hold anything: select, do not multiply
              d0 = v0 ? d0 : 0.f;
              d1 = v1 ? d1 : 0.f;
            }
            pk[c >> 1] = bf16x2_bits(p0, p1);
            dk[c >> 1] = bf16x2_bits(d0, d1);
          }
        }
      };
      if (__shfl_sync(0xffffffffu, qbase, 31) >= 0 && qlim >= 32) pass(std::false_type{});
      else pass(std::true_type{});
      // the MMAs of step i-2 must be done with buffer i & 1 before it is rewritten
      const int pb = i & 1;
      if (i >= 2 && !warp_wait(&mm_done[pb], ((i >> 1) & 1) ^ 1u, abort_flag, status)) { ok = false; break; }
      tc_fence_after();
      tmem_st16(t_p + pb * 32 + half * 16 + lane_off, pk);
      uint8_t* ds = DSs + pb * SLAB;
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const int chunk = half * 4 + c;
        *reinterpret_cast<uint4*>(ds + swz(r, chunk)) = make_uint4(dk[4 * c], dk[4 * c + 1], dk[4 * c + 2], dk[4 * c + 3]);
      }
      fence_proxy_async();
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&p_ready[pb]);
    }
    if (ok && warp_wait(acc_done, 0, abort_flag, status)) {
      tc_fence_after();
      const bool kvalid = key < len;
      if (half == 0) {
        // dK (times c) with the inverse rotation at the key's position
        const float c = rsqrtf((float)DH);
        const int kpos = row_pos(tok, S, row0 + key);
        bf16* krow = dqkv + (long long)(row0 + key) * ldq + (long long)(H + g) * DH;
#pragma unroll 1
        for (int cc = 0; cc < 2; ++cc) {
          float k1[32], k2[32];
          tmem_ld32(t_dk + cc * 32 + lane_off, k1);
          tmem_ld32(t_dk + 64 + cc * 32 + lane_off, k2);
#pragma unroll
          for (int e = 0; e < 32; ++e) {
            const float p1 = c * k1[e], p2 = c * k2[e];
            float cs = 1.f, sn = 0.f;
            if (rcos) {
              cs = rcos[(size_t)kpos * 64 + cc * 32 + e];
              sn = rsin[(size_t)kpos * 64 + cc * 32 + e];
            }
            k1[e] = p1 * cs + p2 * sn;
            k2[e] = p2 * cs - p1 * sn;
          }
          if (kvalid) {
            st_bf16x32_(krow + cc * 32, k1);
            st_bf16x32_(krow + 64 + cc * 32, k2);
          }
        }
      } else {
        bf16* vrow = dqkv + (long long)(row0 + key) * ldq + (long long)(H + Hkv + g) * DH;
#pragma unroll 1
        for (int cc = 0; cc < DH / 32; ++cc) {
          float u[32];
          tmem_ld32(t_dv + cc * 32 + lane_off, u);
          if (kvalid) st_bf16x32_(vrow + cc * 32, u);
        }
      }
    }
  } else {
    // ------------------------------------------------ dQ (warps 10..13)
    // dQ^T from TMEM -> a [64 x 128] float32 tile in shared memory, added
    // into dq_acc by one bulk tensor reduce per step.
    const int quad = warp & 3;
    const int dd = quad * 32 + lane;  // head dimension of this thread
    const uint32_t lane_off = (uint32_t)(quad * 32) << 16;
    const bool leader = (warp == 10 && lane == 0);
    for (int i = 0; i < n_it; ++i) {
      const int h = g * grp + i / (nq - q0), qt = q0 + i % (nq - q0);
      if (!warp_wait(&mm_done[i & 1], (i >> 1) & 1, abort_flag, status)) break;
      tc_fence_after();
      float t0[32], t1[32];
      tmem_ld32(t_dq + lane_off, t0);
      tmem_ld32(t_dq + 32 + lane_off, t1);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(dq_free);
      if (leader && i > 0) bulk_wait_read();  // the previous reduce has read the tile
      named_barrier(1, 128);
#pragma unroll
      for (int e = 0; e < 32; ++e) dqs[e * DH + dd] = t0[e];
#pragma unroll
      for (int e = 0; e < 32; ++e) dqs[(32 + e) * DH + dd] = t1[e];
      fence_proxy_async();
      named_barrier(1, 128);
      if (leader) {
        tma_reduce_add_2d(&tmdq, h * DH, row0 + qt * 64, dqs);
        bulk_commit();
      }
    }
    if (leader) bulk_wait_all();
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

template <bool ALIBI>
cudaError_t bwd_tc(const bf16* qkv, int ldq, const bf16* dO, int ldo, const float* lse, const float* Dvec,
                   float* dq_acc, bf16* dqkv, const int* cnt, int S, int H, int Hkv, int max_seqs, const float* rcos,
                   const float* rsin, const float* alibi, const int* seg, const int* tok, int* status,
                   cudaStream_t st) {
  // K, V, 2 x dS^T (6 slabs) + 3 stages of Q, dO (12 half slabs) + lse/D
  // vectors + dQ staging + alignment + barriers = 232,288 bytes (of 232,448)
  constexpr size_t smem = 6 * SLAB + 12 * HSLAB + 3 * 136 * 4 + 64 * 128 * 4 + 1024 + 256;
  // once per process (initialisation of a function-local static is thread-safe)
  static const cudaError_t attr =
      cudaFuncSetAttribute(attn_bwd_tc_kernel<ALIBI>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (attr != cudaSuccess) return attr;
  CUtensorMap tkv, tq, to, tdq;  // K/V tiles of 128 rows; Q / dO tiles of 64 rows; dQ reduce boxes
  if (!make_map_f32(&tdq, dq_acc, (uint64_t)H * 128, (uint64_t)max_seqs * S, (uint64_t)H * 128, 128, 64))
    return cudaErrorInvalidValue;
  if (!make_map(&tkv, qkv, (uint64_t)ldq, (uint64_t)max_seqs * S, (uint64_t)ldq, 64, 128)) return cudaErrorInvalidValue;
  if (!make_map(&tq, qkv, (uint64_t)ldq, (uint64_t)max_seqs * S, (uint64_t)ldq, 64, 64)) return cudaErrorInvalidValue;
  if (!make_map(&to, dO, (uint64_t)ldo, (uint64_t)max_seqs * S, (uint64_t)ldo, 64, 64)) return cudaErrorInvalidValue;
  // grid (kv head, key tile, sequence): one sequence's blocks are dispatched
  // together, heaviest key tiles (kt = 0) first, so the dQ rows being
  // reduced into at a time are one sequence's (64 MB at the Llama-3-8B
  // shape, inside L2) rather than every kept sequence's
  dim3 grid(Hkv, S / 128, max_seqs);
  attn_bwd_tc_kernel<ALIBI><<<grid, 448, smem, st>>>(tkv, tq, to, tdq, lse, Dvec, max_seqs * S, dq_acc, dqkv, ldq, cnt, S,
                                                     H, Hkv, rcos, rsin, alibi, seg, tok, status);
  return cudaGetLastError();
}
// Backward, head size 64, in two kernels without atomics.
//
// attn_bwd_kv_kernel: dK and dV.  One CTA per (128-key tile, kv head, kept
// sequence); it loops over the query heads of the group and, for each, the
// 128-query tiles at or after the key tile (one step per query tile).  Every
// MMA is M = 128, N = 128.  320 threads:
//   warp 0      TMA: K, V once; Q_i (three stages) and dO_i (one); all lanes
//               write the bf16 terms of -lse_i sqrt(Dh) and -D_i that two
//               extra K = 16 MMAs fold into S^T_i and dP^T_i
//   warp 1      TMEM allocation and the MMAs, issued in the order
//                 dP^T_i, dV += P^T_i dO_i, S^T_{i+1}, dK += dS^T_i Q_i
//               (S^T_0 first): S^T_{i+1} goes ahead of dK_i, so the
//               exponentials of step i+1 overlap dK_i and dP^T_{i+1}
//   warps 2..9  softmax, one key and 64 queries per thread (two warps per
//               TMEM lane quadrant).  Phase A: P^T = exp2(S^T c) written as
//               bf16 over the thread's own S^T columns (the A operand of dV).
//               Phase B: dS^T = P^T (dP^T - D) written as bf16 over its own
//               dP^T columns (the A operand of dK).  At the end dK (times c,
//               with the inverse rotation) and dV from TMEM to dqkv
// TMEM columns: S^T / P^T 0-127, dP^T / dS^T 128-255, dV 256-383, dK 384-511.
// The exponent of P is c S - lse log2(e) = c (S - lse sqrt(Dh)) with
// c = log2(e) / sqrt(Dh), so S^T arrives as S^T - lse sqrt(Dh) and dP^T as
// dP^T - D, and the softmax warps read no per-query vectors.
//
// attn_bwd_q_kernel: dQ.  One CTA per (128-query tile, query head, kept
// sequence), looping over the key tiles at or before the query tile; dQ
// accumulates in TMEM over the loop and is written once, scaled and with the
// inverse rotation, as bf16 (no float32 buffer, no reductions).
// Every MMA has M = 128 (at head size 64 the transposed dQ of the single
// kernel above would be an M = 64 product); the second kernel recomputes S
// and dP (7 MMAs per tile pair, not 5).  At head size 128 the same pair of
// kernels measured slower than the single kernel (95 against 80 ms of
// attention in the Llama-3-8B step), so they serve head size 64 only.

// x as three bf16 terms, t0 + t1 + t2 = x to about 2^-24 |x| (each residual
// is exact in float32).
__device__ __forceinline__ void split3_bf16(float x, uint32_t& t0, uint32_t& t1, uint32_t& t2) {
  const bf16 a = __float2bfloat16_rn(x);
  const float r1 = x - __bfloat162float(a);
  const bf16 b = __float2bfloat16_rn(r1);
  const float r2 = r1 - __bfloat162float(b);
  const bf16 c = __float2bfloat16_rn(r2);
  t0 = __bfloat16_as_ushort(a);
  t1 = __bfloat16_as_ushort(b);
  t2 = __bfloat16_as_ushort(c);
}

template <int DH, bool ALIBI>
__global__ void __launch_bounds__(320, 1)
    attn_bwd_kv_kernel(const __grid_constant__ CUtensorMap tmkv, const __grid_constant__ CUtensorMap tmo,
                       const float* __restrict__ lse, const float* __restrict__ Dvec, int lse_ld,
                       bf16* __restrict__ dqkv, int ldq, const int* __restrict__ cnt,
                       int S, int H, int Hkv, const float* __restrict__ rcos, const float* __restrict__ rsin,
                       const float* __restrict__ alibi, const int* __restrict__ seg, const int* __restrict__ tok,
                       int* status) {
  constexpr int NSL = DH / 64;           // 64-column slabs of a row
  constexpr uint32_t TILE = NSL * SLAB;  // 128 rows x DH bf16
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* Ks = smem;
  uint8_t* Vs = Ks + TILE;
  uint8_t* Qs = Vs + TILE;       // [3] stages: Q_i is read by S^T_i and, a step later, by dK
  uint8_t* dOs = Qs + 3 * TILE;  // one stage
  // XT: 128 rows x 128 bytes (128-byte swizzle) of K = 16 chunk pairs for
  // the fold MMAs: pair 0 = (1, 1, 1, 0, ...) and pair 1 = (0, 0, 0, 1, 1,
  // 1, 0, ...) in every row (the A operands), pair 2 + s = the terms of
  // stage s in row q = query q of the step: (l0, l1, l2, d0, d1, d2, 0, ...)
  // with l0 + l1 + l2 = -lse sqrt(Dh) and d0 + d1 + d2 = -D.
  // (stage 2's terms are pair 0 of a second such slab, XT + SLAB)
  uint8_t* XT = dOs + TILE;
  uint64_t* bars = reinterpret_cast<uint64_t*>(XT + 2 * SLAB);
  uint64_t* kv_full = bars;
  uint64_t* q_full = bars + 1;   // [3]
  uint64_t* q_empty = bars + 4;  // [3]
  uint64_t* o_full = bars + 7;
  uint64_t* o_empty = bars + 8;
  uint64_t* s_full = bars + 9;
  uint64_t* dp_full = bars + 10;
  uint64_t* p_ready = bars + 11;
  uint64_t* ds_ready = bars + 12;
  uint64_t* acc_done = bars + 13;
  uint64_t* drain = bars + 14;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 15);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  // rows row0 .. row0+len-1 (a kept sequence, or with `seg` the kept tokens
  // of sequence blockIdx.z); queries past len get P = dS = 0, keys past len
  // are never stored.  Grid (kv head, key tile, sequence): one sequence's
  // blocks are dispatched together, heaviest key tiles (kt = 0) first.
  const int seq = blockIdx.z;
  int row0, len;
  if (seg) {
    row0 = seg[seq];
    len = seg[seq + 1] - row0;
  } else {
    if (seq >= *cnt) return;
    row0 = seq * S;
    len = S;
  }
  const int kt = blockIdx.y, g = blockIdx.x, grp = H / Hkv;
  if (kt * 128 >= len) return;
  const int nq = (len + 127) / 128;  // query tiles kt .. nq-1 overlap or follow the keys
  const int nqs = nq - kt;
  const int n_it = grp * nqs;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    mbar_init(kv_full, 1);
    for (int s = 0; s < 3; ++s) {
      mbar_init(&q_full[s], 1);
      mbar_init(&q_empty[s], 1);
    }
    mbar_init(o_full, 1);
    mbar_init(o_empty, 1);
    mbar_init(s_full, 1);
    mbar_init(dp_full, 1);
    mbar_init(p_ready, 8);
    mbar_init(ds_ready, 8);
    mbar_init(acc_done, 1);
    mbar_init(drain, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (threadIdx.x < 128) {
    // row r of XT: the two ones patterns, zero terms
    const int r = threadIdx.x;
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      uint4 v = make_uint4(0u, 0u, 0u, 0u);
      if (u == 0) v = make_uint4(0x3F803F80u, 0x3F80u, 0u, 0u);
      if (u == 2) v = make_uint4(0u, 0x3F800000u, 0x3F803F80u, 0u);
      *reinterpret_cast<uint4*>(XT + swz(r, u)) = v;
      *reinterpret_cast<uint4*>(XT + SLAB + swz(r, u)) = make_uint4(0u, 0u, 0u, 0u);
    }
    fence_proxy_async();
  }
  if (warp == 1) tmem_alloc(tmem_slot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t t_s = tmem, t_dp = tmem + 128, t_dv = tmem + 256, t_dk = tmem + 384;

  if (warp == 0) {
    // ------------------------------------------------ producer (warp 0)
    const int kcol = (H + g) * DH, vcol = (H + Hkv + g) * DH;
    if (lane == 0) {
      mbar_arrive_expect_tx(kv_full, 2 * TILE);
      for (int c = 0; c < NSL; ++c) {
        tma_load_2d(Ks + c * SLAB, &tmkv, kcol + 64 * c, row0 + kt * 128, kv_full);
        tma_load_2d(Vs + c * SLAB, &tmkv, vcol + 64 * c, row0 + kt * 128, kv_full);
      }
    }
    const float sq_dh = sqrtf((float)DH);
    // -lse sqrt(Dh) and -D of the 128 queries of step i, four a lane, loaded
    // one step ahead so their latency stays off the Q copy's path
    float xl[4], xd[4];
    auto load_terms = [&](int i) {
      const int h = g * grp + i / nqs, qt = kt + i % nqs;
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int q = u * 32 + lane;
        xl[u] = 0.f;
        xd[u] = 0.f;
        if (qt * 128 + q < len) {
          const size_t at = (size_t)h * lse_ld + row0 + qt * 128 + q;
          xl[u] = -lse[at] * sq_dh;
          xd[u] = -Dvec[at];
        }
      }
    };
    if (n_it > 0) load_terms(0);
    int nql = 0, nol = 0;
    for (int i = 0; i < n_it; ++i) {
      const int s = i % 3;
      const int h = g * grp + i / nqs, qt = kt + i % nqs;
      // Q_i and the terms of step i into stage s once step i-3 has released
      // it; the copy is issued first (the barrier's phase cannot complete
      // before the arrival below, which follows the terms)
      if (!warp_wait(&q_empty[s], ((i / 3) & 1) ^ 1u, abort_flag, status)) break;
      if (lane == 0)
        for (int c = 0; c < NSL; ++c)
          tma_load_2d(Qs + s * TILE + c * SLAB, &tmkv, h * DH + 64 * c, row0 + qt * 128, &q_full[s]);
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        uint32_t l0, l1, l2, d0, d1, d2;
        split3_bf16(xl[u], l0, l1, l2);
        split3_bf16(xd[u], d0, d1, d2);
        *reinterpret_cast<uint4*>(s < 2 ? XT + swz(u * 32 + lane, 4 + 2 * s) : XT + SLAB + swz(u * 32 + lane, 0)) =
            make_uint4(l0 | (l1 << 16), l2 | (d0 << 16), d1 | (d2 << 16), 0u);
      }
      fence_proxy_async();
      __syncwarp();
      if (lane == 0) mbar_arrive_expect_tx(&q_full[s], TILE);
      if (i + 1 < n_it) load_terms(i + 1);
      ++nql;
      // dO_i once dV_{i-1} has read dO_{i-1}
      if (!warp_wait(o_empty, (i & 1) ^ 1u, abort_flag, status)) break;
      if (lane == 0) {
        mbar_arrive_expect_tx(o_full, TILE);
        for (int c = 0; c < NSL; ++c)
          tma_load_2d(dOs + c * SLAB, &tmo, h * DH + 64 * c, row0 + qt * 128, o_full);
      }
      ++nol;
    }
    if (lane == 0 && *abort_flag) {
      // let every copy in flight land before the block exits
      mbar_drain(kv_full, 0);
      for (int i = nql > 3 ? nql - 3 : 0; i < nql; ++i) mbar_drain(&q_full[i % 3], (i / 3) & 1);
      if (nol > 0) mbar_drain(o_full, (nol - 1) & 1);
    }
    __syncwarp();
  } else if (warp == 1) {
    {  // the whole warp, converged; one elected lane issues
      // ------------------------------------------------ MMA issuer
      constexpr uint32_t ID_S = idesc_bf16(128, 128, false, false);   // S^T, dP^T and the folds
      constexpr uint32_t ID_KV = idesc_bf16(128, DH, false, true);    // dV, dK (B = dO / Q, MN-major)
      // shared-memory descriptors built once; an MMA's operand is its base
      // plus (byte offset >> 4) in the address field (every tile lies below
      // 256 KB, so the 14-bit field never carries)
      const uint64_t DK = sdesc(smem_u32(Ks), 16, 1024), DV = sdesc(smem_u32(Vs), 16, 1024);
      const uint64_t DQ = sdesc(smem_u32(Qs), 16, 1024), DO = sdesc(smem_u32(dOs), 16, 1024);
      const uint64_t DQMN = sdesc(smem_u32(Qs), SLAB, 1024), DOMN = sdesc(smem_u32(dOs), SLAB, 1024);
      const uint64_t DX = sdesc(smem_u32(XT), 16, 1024), DX2 = sdesc(smem_u32(XT + SLAB), 16, 1024);
      // B operand of the fold MMAs: the terms of Q stage s
      auto terms = [&](int s) { return s < 2 ? DX + (uint64_t)(((2 + s) * 32) >> 4) : DX2; };
      // offset of the K = 16 chunk kk of a K-major 128 x 128 tile (two slabs)
      auto kmaj = [](int kk) { return (uint64_t)(((kk >> 2) * SLAB + (kk & 3) * 32) >> 4); };
      // S^T_i = K Q_i^T - lse sqrt(Dh) (ones pattern 0 times the terms)
      auto issue_s = [&](int i) -> bool {
        const int s = i % 3;
        if (!mbar_wait_conv(&q_full[s], (i / 3) & 1, abort_flag, status)) return false;
        tc_fence_after();
        const uint64_t st = (uint64_t)((s * TILE) >> 4);
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk) mma_bf16_w(t_s, DK + kmaj(kk), DQ + st + kmaj(kk), ID_S, kk > 0);
        mma_bf16_w(t_s, DX, terms(s), ID_S, 1u);
        mma_commit_w(s_full);
        return true;
      };
      bool ok = mbar_wait_conv(kv_full, 0, abort_flag, status) && issue_s(0);
      for (int i = 0; ok && i < n_it; ++i) {
        const int s = i % 3;
        const uint64_t st = (uint64_t)((s * TILE) >> 4);
        // dP^T_i = V dO_i^T - D (ones pattern 1 times the terms), over the
        // dS^T_{i-1} columns (dK_{i-1}, issued before, reads them first)
        if (!mbar_wait_conv(o_full, i & 1, abort_flag, status)) { ok = false; break; }
        tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk) mma_bf16_w(t_dp, DV + kmaj(kk), DO + kmaj(kk), ID_S, kk > 0);
        mma_bf16_w(t_dp, DX + (uint64_t)(32 >> 4), terms(s), ID_S, 1u);
        mma_commit_w(dp_full);
        // dV += P^T_i dO_i: A = P^T from TMEM (queries 64h..64h+63 as bf16
        // pairs in columns 64h..64h+31), B = dO MN-major
        if (!mbar_wait_conv(p_ready, i & 1, abort_flag, status)) { ok = false; break; }
        tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < 8; ++kk)
          mma_bf16_ta_w(t_dv, t_s + 64 * (kk >> 2) + 8 * (kk & 3), DOMN + (uint64_t)((kk * 2048) >> 4), ID_KV,
                      (i > 0 || kk > 0) ? 1u : 0u);
        mma_commit_w(o_empty);
        // S^T_{i+1} ahead of the product that waits for dS^T_i
        if (i + 1 < n_it && !issue_s(i + 1)) { ok = false; break; }
        if (!mbar_wait_conv(ds_ready, i & 1, abort_flag, status)) { ok = false; break; }
        tc_fence_after();
        // dK += dS^T_i Q_i (contraction over the 128 queries): A = dS^T from
        // TMEM (queries 64h..64h+63 as bf16 pairs in dP^T columns
        // 64h..64h+31), B = Q MN-major
#pragma unroll
        for (int kk = 0; kk < 8; ++kk)
          mma_bf16_ta_w(t_dk, t_dp + 64 * (kk >> 2) + 8 * (kk & 3), DQMN + st + (uint64_t)((kk * 2048) >> 4), ID_KV,
                      (i > 0 || kk > 0) ? 1u : 0u);
        mma_commit_w(&q_empty[s]);
      }
      if (ok) {
        mma_commit_w(acc_done);
      } else {
        mma_commit_w(drain);
        if (lane == 0) mbar_drain(drain, 0);
        __syncwarp();
      }
    }
  } else {
    // ------------------------------------------------ P / dS (warps 2..9)
    // two warps per TMEM lane quadrant: warps 2..5 take queries 0..63 of the
    // step, warps 6..9 queries 64..127, one key per thread
    const int quad = warp & 3;
    const int half = (warp - 2) >> 2;
    const int r = quad * 32 + lane;  // key within the tile
    const int key = kt * 128 + r;
    const uint32_t lane_off = (uint32_t)(quad * 32) << 16;
    const uint32_t t_sh = t_s + half * 64 + lane_off, t_dph = t_dp + half * 64 + lane_off;
    const float sl2 = kLog2e * rsqrtf((float)DH);
    bool ok = true;
    for (int i = 0; i < n_it; ++i) {
      const int qt = kt + i % nqs;
      // ALiBi: logit bias slope2 (key - query) of this step's query head
      const float slope2 = ALIBI ? alibi[g * grp + i / nqs] * kLog2e : 0.f;
      const int qbase = qt * 128 + half * 64 - key;  // query c is visible iff qbase + c >= 0
      const int qlim = len - (qt * 128 + half * 64);  // and exists iff c < qlim (warp-uniform)
      // mask only where some of the warp's 32 keys do not see all 64 queries,
      // or the queries run past the sequence (warp-uniform)
      const bool full = __shfl_sync(0xffffffffu, qbase, 31) >= 0 && qlim >= 64;
      // ---- phase A: P^T from S^T (lse folded in)
      if (!warp_wait(s_full, i & 1, abort_flag, status)) { ok = false; break; }
      tc_fence_after();
      uint32_t pk[32];
      auto phase_a = [&](auto masked) {
        constexpr bool MASK = decltype(masked)::value;
        const uint64_t sl2x2 = f2_pack(sl2, sl2);
        const float b0 = slope2 * (float)(-qbase);  // bias of query c: b0 - slope2 c
        const uint64_t nsx2 = f2_pack(-slope2, -slope2), b0x2 = f2_pack(b0, b0);
        uint32_t sr[2][32];
        tmem_ld32_nw(t_sh, sr[0]);
        tmem_ld32_nw(t_sh + 32, sr[1]);
        tmem_wait_ld();
#pragma unroll
        for (int h2 = 0; h2 < 2; ++h2) {
#pragma unroll
          for (int c2 = 0; c2 < 32; c2 += 2) {
            const int c = h2 * 32 + c2;
            uint64_t x2 = f2_mul(f2_pack(__uint_as_float(sr[h2][c2]), __uint_as_float(sr[h2][c2 + 1])), sl2x2);
            if constexpr (ALIBI) x2 = f2_add(x2, f2_fma(f2_pack((float)c, (float)(c + 1)), nsx2, b0x2));
            float x0, x1;
            f2_unpack(x2, x0, x1);
            float p0 = ex2(x0), p1 = ex2(x1);
            if constexpr (MASK) {
              p0 = (qbase + c >= 0 && c < qlim) ? p0 : 0.f;
              p1 = (qbase + c + 1 >= 0 && c + 1 < qlim) ? p1 : 0.f;
            }
            pk[c >> 1] = bf16x2_bits(p0, p1);
          }
        }
      };
      if (full) phase_a(std::false_type{});
      else phase_a(std::true_type{});
      // P^T (queries 64 half .. 64 half + 63) over this warp's own S^T columns
      tmem_st32u(t_sh, pk);
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(p_ready);
      // ---- phase B: dS^T = P^T (dP^T - D) (D folded in)
      if (!warp_wait(dp_full, i & 1, abort_flag, status)) { ok = false; break; }
      tc_fence_after();
      // dS^T over the packed P^T in place (pk), both halves loaded at once
      uint32_t dr[2][32];
      tmem_ld32_nw(t_dph, dr[0]);
      tmem_ld32_nw(t_dph + 32, dr[1]);
      tmem_wait_ld();
#pragma unroll
      for (int h2 = 0; h2 < 2; ++h2) {
#pragma unroll
        for (int c2 = 0; c2 < 32; c2 += 2) {
          const uint32_t pw = pk[(h2 * 32 + c2) >> 1];
          const uint64_t pp = f2_pack(__uint_as_float(pw << 16), __uint_as_float(pw & 0xFFFF0000u));
          float d0, d1;
          f2_unpack(f2_mul(pp, f2_pack(__uint_as_float(dr[h2][c2]), __uint_as_float(dr[h2][c2 + 1]))), d0, d1);
          if (!full) {  // rows past the sequence may hold anything: select, do not multiply
            const int c = h2 * 32 + c2;
            d0 = (qbase + c >= 0 && c < qlim) ? d0 : 0.f;
            d1 = (qbase + c + 1 >= 0 && c + 1 < qlim) ? d1 : 0.f;
          }
          pk[(h2 * 32 + c2) >> 1] = bf16x2_bits(d0, d1);
        }
      }
      // dS^T (queries 64 half .. 64 half + 63) over this warp's own dP^T columns
      tmem_st32u(t_dph, pk);
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(ds_ready);
    }
    if (ok && warp_wait(acc_done, 0, abort_flag, status)) {
      tc_fence_after();
      const bool kvalid = key < len;
      if (half == 0) {
        // dK (times c) with the inverse rotation at the key's position
        const float c = rsqrtf((float)DH);
        const int kpos = kvalid ? row_pos(tok, S, row0 + key) : 0;  // rows past the segment are not read
        bf16* krow = dqkv + (long long)(row0 + key) * ldq + (long long)(H + g) * DH;
#pragma unroll 1
        for (int cc = 0; cc < DH / 64; ++cc) {
          float k1[32], k2[32];
          tmem_ld32(t_dk + cc * 32 + lane_off, k1);
          tmem_ld32(t_dk + DH / 2 + cc * 32 + lane_off, k2);
#pragma unroll
          for (int e = 0; e < 32; ++e) {
            const float p1 = c * k1[e], p2 = c * k2[e];
            float cs = 1.f, sn = 0.f;
            if (rcos) {
              cs = rcos[(size_t)kpos * (DH / 2) + cc * 32 + e];
              sn = rsin[(size_t)kpos * (DH / 2) + cc * 32 + e];
            }
            k1[e] = p1 * cs + p2 * sn;
            k2[e] = p2 * cs - p1 * sn;
          }
          if (kvalid) {
            st_bf16x32_(krow + cc * 32, k1);
            st_bf16x32_(krow + DH / 2 + cc * 32, k2);
          }
        }
      } else {
        bf16* vrow = dqkv + (long long)(row0 + key) * ldq + (long long)(H + Hkv + g) * DH;
#pragma unroll 1
        for (int cc = 0; cc < DH / 32; ++cc) {
          float u[32];
          tmem_ld32(t_dv + cc * 32 + lane_off, u);
          if (kvalid) st_bf16x32_(vrow + cc * 32, u);
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// dQ of one (128-query tile, query head h, kept sequence): for each key tile
// j <= qt, S_j = Q K_j^T and dP_j = dO V_j^T (M = 128 queries, N = 128 keys),
// dS_j = P_j (dP_j - D) with P_j = exp2(S_j c - lse log2 e), and
// dQ += dS_j K_j.  320 threads:
//   warp 0      TMA: Q and dO once, then K_j (three stages) and V_j (two)
//   warp 1      TMEM allocation and the MMAs, in the order S_0, dP_0, then
//               per step S_{j+1}, dQ += dS_j K_j, dP_{j+1}: S is double-
//               buffered, so S_{j+1} runs while the softmax works on step j
//   warps 2..9  softmax, one query row and 64 keys per thread (two warps per
//               TMEM lane quadrant), lse and D of the row held in registers:
//               P_j from S_j, then dS_j from dP_j, written as bf16 over the
//               thread's own S_j columns (the A operand of dQ += dS_j K_j);
//               at the end dQ (times c, with the inverse rotation at the
//               query's position) from TMEM to dqkv
// TMEM columns: S_0 0-127, S_1 128-255, dP 256-383, dQ 384-511.
template <int DH, bool ALIBI>
__global__ void __launch_bounds__(320, 1)
    attn_bwd_q_kernel(const __grid_constant__ CUtensorMap tmkv, const __grid_constant__ CUtensorMap tmo,
                      const float* __restrict__ lse, const float* __restrict__ Dvec, int lse_ld,
                      bf16* __restrict__ dqkv, int ldq, const int* __restrict__ cnt, int S, int H, int Hkv,
                      const float* __restrict__ rcos, const float* __restrict__ rsin,
                      const float* __restrict__ alibi, const int* __restrict__ seg, const int* __restrict__ tok,
                      int* status) {
  constexpr int NSL = DH / 64;           // 64-column slabs of a row
  constexpr uint32_t TILE = NSL * SLAB;  // 128 rows x DH bf16
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* Qs = smem;
  uint8_t* dOs = Qs + TILE;
  uint8_t* Ks = dOs + TILE;      // [3] stages: K_j is read by S_j and, a step later, by dQ
  uint8_t* Vs = Ks + 3 * TILE;   // [2] stages
  uint64_t* bars = reinterpret_cast<uint64_t*>(Vs + 2 * TILE);
  uint64_t* qo_full = bars;
  uint64_t* k_full = bars + 1;   // [3]
  uint64_t* k_empty = bars + 4;  // [3]
  uint64_t* v_full = bars + 7;   // [2]
  uint64_t* v_empty = bars + 9;  // [2]
  uint64_t* s_full = bars + 11;  // [2] per S buffer
  uint64_t* dp_full = bars + 13;
  uint64_t* ds_ready = bars + 14;
  uint64_t* acc_done = bars + 15;
  uint64_t* drain = bars + 16;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 17);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  // rows row0 .. row0+len-1 as in the forward; query rows past len are not
  // stored (P = dS = 0 for them), keys past len are hidden by causality.
  // Grid (query head, query tile, sequence), heaviest query tiles first.
  const int seq = blockIdx.z;
  int row0, len;
  if (seg) {
    row0 = seg[seq];
    len = seg[seq + 1] - row0;
  } else {
    if (seq >= *cnt) return;
    row0 = seq * S;
    len = S;
  }
  const int qt = (int)gridDim.y - 1 - (int)blockIdx.y;
  if (qt * 128 >= len) return;
  const int h = blockIdx.x, g = (h * Hkv) / H;
  // key tiles qt, qt-1, .., 0 (step j takes tile qt - j): the blocks of a
  // head group then fetch different K / V tiles at a time
  const int n_k = qt + 1;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    mbar_init(qo_full, 1);
    for (int s = 0; s < 3; ++s) {
      mbar_init(&k_full[s], 1);
      mbar_init(&k_empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&v_full[s], 1);
      mbar_init(&v_empty[s], 1);
      mbar_init(&s_full[s], 1);
    }
    mbar_init(dp_full, 1);
    mbar_init(ds_ready, 8);
    mbar_init(acc_done, 1);
    mbar_init(drain, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(tmem_slot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t t_dp = tmem + 256, t_dq = tmem + 384;

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------ TMA producer
      const int kcol = (H + g) * DH, vcol = (H + Hkv + g) * DH;
      mbar_arrive_expect_tx(qo_full, 2 * TILE);
      for (int c = 0; c < NSL; ++c) {
        tma_load_2d(Qs + c * SLAB, &tmkv, h * DH + 64 * c, row0 + qt * 128, qo_full);
        tma_load_2d(dOs + c * SLAB, &tmo, h * DH + 64 * c, row0 + qt * 128, qo_full);
      }
      int nkl = 0, nvl = 0;
      for (int j = 0; j < n_k; ++j) {
        const int s = j & 1, sk = j % 3;
        if (!mbar_wait(&k_empty[sk], ((j / 3) & 1) ^ 1u, abort_flag, status)) break;
        mbar_arrive_expect_tx(&k_full[sk], TILE);
        for (int c = 0; c < NSL; ++c)
          tma_load_2d(Ks + sk * TILE + c * SLAB, &tmkv, kcol + 64 * c, row0 + (qt - j) * 128, &k_full[sk]);
        ++nkl;
        if (!mbar_wait(&v_empty[s], ((j >> 1) & 1) ^ 1u, abort_flag, status)) break;
        mbar_arrive_expect_tx(&v_full[s], TILE);
        for (int c = 0; c < NSL; ++c)
          tma_load_2d(Vs + s * TILE + c * SLAB, &tmkv, vcol + 64 * c, row0 + (qt - j) * 128, &v_full[s]);
        ++nvl;
      }
      if (*abort_flag) {
        // let every copy in flight land before the block exits
        mbar_drain(qo_full, 0);
        for (int j = nkl > 3 ? nkl - 3 : 0; j < nkl; ++j) mbar_drain(&k_full[j % 3], (j / 3) & 1);
        for (int j = nvl > 2 ? nvl - 2 : 0; j < nvl; ++j) mbar_drain(&v_full[j & 1], (j >> 1) & 1);
      }
    }
  } else if (warp == 1) {
    {  // the whole warp, converged; one elected lane issues
      // ------------------------------------------------ MMA issuer
      constexpr uint32_t ID_S = idesc_bf16(128, 128, false, false);  // S, dP (both operands K-major)
      constexpr uint32_t ID_Q = idesc_bf16(128, DH, false, true);    // dQ (A = dS from TMEM, B = K MN-major)
      const uint64_t DQ = sdesc(smem_u32(Qs), 16, 1024), DO = sdesc(smem_u32(dOs), 16, 1024);
      const uint64_t DK = sdesc(smem_u32(Ks), 16, 1024), DV = sdesc(smem_u32(Vs), 16, 1024);
      const uint64_t DKMN = sdesc(smem_u32(Ks), SLAB, 1024);
      auto kmaj = [](int kk) { return (uint64_t)(((kk >> 2) * SLAB + (kk & 3) * 32) >> 4); };
      // S_j = Q K_j^T into S buffer j & 1
      auto issue_s = [&](int j) -> bool {
        const int s = j & 1, sk = j % 3;
        if (!mbar_wait_conv(&k_full[sk], (j / 3) & 1, abort_flag, status)) return false;
        tc_fence_after();
        const uint64_t st = (uint64_t)((sk * TILE) >> 4);
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk) mma_bf16_w(tmem + s * 128, DQ + kmaj(kk), DK + st + kmaj(kk), ID_S, kk > 0);
        mma_commit_w(&s_full[s]);
        return true;
      };
      // dP_j = dO V_j^T
      auto issue_dp = [&](int j) -> bool {
        const int s = j & 1;
        if (!mbar_wait_conv(&v_full[s], (j >> 1) & 1, abort_flag, status)) return false;
        tc_fence_after();
        const uint64_t st = (uint64_t)((s * TILE) >> 4);
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk) mma_bf16_w(t_dp, DO + kmaj(kk), DV + st + kmaj(kk), ID_S, kk > 0);
        mma_commit_w(dp_full);
        mma_commit_w(&v_empty[s]);
        return true;
      };
      bool ok = mbar_wait_conv(qo_full, 0, abort_flag, status) && issue_s(0) && issue_dp(0);
      for (int j = 0; ok && j < n_k; ++j) {
        const int s = j & 1;
        // S_{j+1} into the other buffer (its dS_{j-1} was read by dQ, issued before)
        if (j + 1 < n_k && !issue_s(j + 1)) { ok = false; break; }
        // dQ += dS_j K_j: A = dS_j from TMEM (keys 64h..64h+63 as bf16 pairs
        // in columns 64h..64h+31 of S buffer s), B = K_j MN-major
        if (!mbar_wait_conv(ds_ready, j & 1, abort_flag, status)) { ok = false; break; }
        tc_fence_after();
        const uint64_t sk = (uint64_t)(((j % 3) * TILE) >> 4);
#pragma unroll
        for (int kk = 0; kk < 8; ++kk)
          mma_bf16_ta_w(t_dq, tmem + s * 128 + 64 * (kk >> 2) + 8 * (kk & 3), DKMN + sk + (uint64_t)((kk * 2048) >> 4),
                      ID_Q, (j > 0 || kk > 0) ? 1u : 0u);
        mma_commit_w(&k_empty[j % 3]);
        // dP_{j+1} over dP_j, which the softmax warps have read (ds_ready)
        if (j + 1 < n_k && !issue_dp(j + 1)) { ok = false; break; }
      }
      if (ok) {
        mma_commit_w(acc_done);
      } else {
        mma_commit_w(drain);
        if (lane == 0) mbar_drain(drain, 0);
        __syncwarp();
      }
    }
  } else {
    // ------------------------------------------------ softmax (warps 2..9)
    // two warps per TMEM lane quadrant: warps 2..5 take keys 0..63 of each
    // key tile, warps 6..9 keys 64..127, one query row per thread
    const int quad = warp & 3;
    const int half = (warp - 2) >> 2;
    const int r = quad * 32 + lane;  // query row within the tile
    const int q = qt * 128 + r;      // query within the sequence
    const bool qvalid = q < len;
    const uint32_t lane_off = (uint32_t)(quad * 32) << 16;
    const float sl2 = kLog2e * rsqrtf((float)DH);
    const float slope2 = ALIBI ? alibi[h] * kLog2e : 0.f;
    float lse2 = 0.f, dq = 0.f;  // lse log2(e) and D of this row
    if (qvalid) {
      const size_t at = (size_t)h * lse_ld + row0 + q;
      lse2 = lse[at] * kLog2e;
      dq = Dvec[at];
    }
    // rows past the sequence: P = dS = 0 (warp-uniform test below)
    const bool any_invalid = __any_sync(0xffffffffu, !qvalid);
    bool ok = true;
    for (int j = 0; j < n_k; ++j) {
      const int s = j & 1;
      const uint32_t t_sh = tmem + s * 128 + half * 64 + lane_off, t_dph = t_dp + half * 64 + lane_off;
      // key c of this half is visible iff kbase + c <= q
      const int kbase = (qt - j) * 128 + half * 64;
      const bool masked = (j == 0) || any_invalid;  // the diagonal tile comes first (warp-uniform)
      if (!warp_wait(&s_full[s], (j >> 1) & 1, abort_flag, status)) { ok = false; break; }
      tc_fence_after();
      // P = exp2(S c - lse log2 e (+ ALiBi bias)) for 64 keys, kept as bf16 pairs
      uint32_t pk[32];
      {
        const uint64_t sl2x2 = f2_pack(sl2, sl2), nl2 = f2_pack(-lse2, -lse2);
        const float b0 = slope2 * (float)(kbase - q);  // bias of key c: b0 + slope2 c
        const uint64_t sx2 = f2_pack(slope2, slope2), b0x2 = f2_pack(b0, b0);
        uint32_t sr[2][32];
        tmem_ld32_nw(t_sh, sr[0]);
        tmem_ld32_nw(t_sh + 32, sr[1]);
        tmem_wait_ld();
#pragma unroll
        for (int h2 = 0; h2 < 2; ++h2) {
#pragma unroll
          for (int c2 = 0; c2 < 32; c2 += 2) {
            const int c = h2 * 32 + c2;
            uint64_t add = nl2;
            if constexpr (ALIBI) add = f2_add(nl2, f2_fma(f2_pack((float)c, (float)(c + 1)), sx2, b0x2));
            float x0, x1;
            f2_unpack(f2_fma(f2_pack(__uint_as_float(sr[h2][c2]), __uint_as_float(sr[h2][c2 + 1])), sl2x2, add), x0, x1);
            float p0 = ex2(x0), p1 = ex2(x1);
            if (masked) {  // select, do not multiply: rows past the sequence may hold anything
              p0 = (qvalid && kbase + c <= q) ? p0 : 0.f;
              p1 = (qvalid && kbase + c + 1 <= q) ? p1 : 0.f;
            }
            pk[c >> 1] = bf16x2_bits(p0, p1);
          }
        }
      }
      // dS = P (dP - D), written as bf16 pairs over this warp's own S columns
      if (!warp_wait(dp_full, j & 1, abort_flag, status)) { ok = false; break; }
      tc_fence_after();
      {
        // dS over the packed P in place (pk), both halves loaded at once
        const uint64_t nd2 = f2_pack(-dq, -dq);
        uint32_t dr[2][32];
        tmem_ld32_nw(t_dph, dr[0]);
        tmem_ld32_nw(t_dph + 32, dr[1]);
        tmem_wait_ld();
#pragma unroll
        for (int h2 = 0; h2 < 2; ++h2) {
#pragma unroll
          for (int c2 = 0; c2 < 32; c2 += 2) {
            const int c = h2 * 32 + c2;
            const uint32_t pw = pk[c >> 1];
            const uint64_t pp = f2_pack(__uint_as_float(pw << 16), __uint_as_float(pw & 0xFFFF0000u));
            float d0, d1;
            f2_unpack(f2_mul(pp, f2_add(f2_pack(__uint_as_float(dr[h2][c2]), __uint_as_float(dr[h2][c2 + 1])), nd2)),
                      d0, d1);
            if (masked) {
              d0 = (qvalid && kbase + c <= q) ? d0 : 0.f;
              d1 = (qvalid && kbase + c + 1 <= q) ? d1 : 0.f;
            }
            pk[c >> 1] = bf16x2_bits(d0, d1);
          }
        }
      }
      tmem_st32u(t_sh, pk);
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(ds_ready);
    }
    // dQ times c with the inverse rotation at the query's position: this
    // thread takes the pairs (i, i + DH/2), i = off .. off + 31 (head size
    // 64: the first warp of each quadrant alone)
    const int off = DH == 128 ? half * 32 : 0;
    if (ok && warp_wait(acc_done, 0, abort_flag, status) && (DH == 128 || half == 0)) {
      tc_fence_after();
      const float c = rsqrtf((float)DH);
      const int pos = qvalid ? row_pos(tok, S, row0 + q) : 0;
      float a1[32], a2[32];
      tmem_ld32(t_dq + off + lane_off, a1);
      tmem_ld32(t_dq + DH / 2 + off + lane_off, a2);
#pragma unroll
      for (int e = 0; e < 32; ++e) {
        const float p1 = c * a1[e], p2 = c * a2[e];
        float cs = 1.f, sn = 0.f;
        if (rcos) {
          cs = rcos[(size_t)pos * (DH / 2) + off + e];
          sn = rsin[(size_t)pos * (DH / 2) + off + e];
        }
        a1[e] = p1 * cs + p2 * sn;
        a2[e] = p2 * cs - p1 * sn;
      }
      if (qvalid) {
        bf16* qrow = dqkv + (long long)(row0 + q) * ldq + (long long)h * DH;
        st_bf16x32_(qrow + off, a1);
        st_bf16x32_(qrow + DH / 2 + off, a2);
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

template <int DH, bool ALIBI>
cudaError_t bwd_split(const bf16* qkv, int ldq, const bf16* dO, int ldo, const float* lse, const float* Dvec,
                      bf16* dqkv, const int* cnt, int S, int H, int Hkv, int max_seqs, const float* rcos,
                      const float* rsin, const float* alibi, const int* seg, const int* tok, int* status,
                      cudaStream_t st) {
  constexpr size_t TILE = (size_t)(DH / 64) * SLAB;
  // dK / dV: K, V, 3 stages of Q, dO (six tiles) + XT (two slabs) +
  // alignment + barriers
  constexpr size_t smem_kv = 6 * TILE + 2 * SLAB + 1024 + 256;
  // dQ: Q, dO, 3 stages of K, 2 of V (seven tiles) + alignment + barriers
  constexpr size_t smem_q = 7 * TILE + 1024 + 256;
  // once per process (initialisation of a function-local static is thread-safe)
  static const cudaError_t attr = [] {
    cudaError_t e = cudaFuncSetAttribute(attn_bwd_kv_kernel<DH, ALIBI>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem_kv);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(attn_bwd_q_kernel<DH, ALIBI>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               (int)smem_q);
    return e;
  }();
  if (attr != cudaSuccess) return attr;
  CUtensorMap tkv, to;  // tiles of 128 rows x 64 columns: Q, K, V in qkv; dO
  if (!make_map(&tkv, qkv, (uint64_t)ldq, (uint64_t)max_seqs * S, (uint64_t)ldq, 64, 128)) return cudaErrorInvalidValue;
  if (!make_map(&to, dO, (uint64_t)ldo, (uint64_t)max_seqs * S, (uint64_t)ldo, 64, 128)) return cudaErrorInvalidValue;
  attn_bwd_kv_kernel<DH, ALIBI><<<dim3(Hkv, S / 128, max_seqs), 320, smem_kv, st>>>(
      tkv, to, lse, Dvec, max_seqs * S, dqkv, ldq, cnt, S, H, Hkv, rcos, rsin, alibi, seg, tok, status);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  attn_bwd_q_kernel<DH, ALIBI><<<dim3(H, S / 128, max_seqs), 320, smem_q, st>>>(
      tkv, to, lse, Dvec, max_seqs * S, dqkv, ldq, cnt, S, H, Hkv, rcos, rsin, alibi, seg, tok, status);
  return cudaGetLastError();
}
}  // namespace

bool attn_tc_supported(int S, int Dh) { return S % 128 == 0 && (Dh == 64 || Dh == 128); }

bool attn_bwd_tc_supported(int S, int Dh) { return S % 128 == 0 && (Dh == 64 || Dh == 128); }

cudaError_t launch_attn_bwd_tc(const bf16* qkv, int ldqkv, const bf16* dO, int ldo, const float* lse,
                               const float* Dvec, float* dq_acc, bf16* dqkv, const int* cnt, int S, int H, int Hkv,
                               int Dh, int max_seqs, const float* rcos, const float* rsin, const float* alibi,
                               const int* seg, const int* tok, int* status, cudaStream_t st) {
  if (Dh == 64) {  // dQ, dK, dV straight into dqkv (two kernels, no float32 dQ)
    if (alibi)
      return bwd_split<64, true>(qkv, ldqkv, dO, ldo, lse, Dvec, dqkv, cnt, S, H, Hkv, max_seqs, rcos, rsin, alibi,
                                 seg, tok, status, st);
    return bwd_split<64, false>(qkv, ldqkv, dO, ldo, lse, Dvec, dqkv, cnt, S, H, Hkv, max_seqs, rcos, rsin, alibi,
                                seg, tok, status, st);
  }
  cudaError_t e = cudaMemsetAsync(dq_acc, 0, (size_t)max_seqs * S * H * 128 * sizeof(float), st);
  if (e != cudaSuccess) return e;
  e = alibi ? bwd_tc<true>(qkv, ldqkv, dO, ldo, lse, Dvec, dq_acc, dqkv, cnt, S, H, Hkv, max_seqs, rcos, rsin, alibi,
                           seg, tok, status, st)
            : bwd_tc<false>(qkv, ldqkv, dO, ldo, lse, Dvec, dq_acc, dqkv, cnt, S, H, Hkv, max_seqs, rcos, rsin, alibi,
                            seg, tok, status, st);
  if (e != cudaSuccess) return e;
  // dQ from the float32 buffer: scaled and rotated into dqkv
  return launch_dq_finish(dq_acc, dqkv, ldqkv, H, 128, rcos, rsin, cnt, S, max_seqs * S, tok, st);
}

cudaError_t launch_attn_fwd_tc(const bf16* qkv, int ldqkv, bf16* o, int ldo, float* lse, const int* cnt, int S, int H,
                               int Hkv, int Dh, int max_seqs, const float* alibi, const int* seg, int* status,
                               cudaStream_t st) {
  if (Dh == 64) {
    if (alibi) return fwd_tc<64, true>(qkv, ldqkv, o, ldo, lse, cnt, S, H, Hkv, max_seqs, alibi, seg, status, st);
    return fwd_tc<64, false>(qkv, ldqkv, o, ldo, lse, cnt, S, H, Hkv, max_seqs, alibi, seg, status, st);
  }
  if (alibi) return fwd_pp<true>(qkv, ldqkv, o, ldo, lse, cnt, S, H, Hkv, max_seqs, alibi, seg, status, st);
  return fwd_pp<false>(qkv, ldqkv, o, ldo, lse, cnt, S, H, Hkv, max_seqs, alibi, seg, status, st);
}

}  // namespace ldk
