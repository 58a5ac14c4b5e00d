// Layer-dropout masks and kept-sequence lists, all layers in one launch.
//
// Eq. (layer_dropout_train): M^{l,t} in {0,1}^B ~ Bernoulli(1 - p^{l,t});
// Tensor Granularity subsection: one draw per sequence, or one per layer
// and step for the whole batch; Preliminary section: the layer then runs on
// {b : M[b] = 1} only, which this kernel lists in ascending b.  A shard of a
// data-parallel batch draws with its global sequence indices (b_offset + b).
//
// Draw: u = word 0 of Philox4x32-10 (Salmon et al., SC'11) with key
// (seed lo, seed hi) and counter (b', l, t lo, t hi), b' = b per sequence
// 0 per batch and b_offset per shard.  Sequence b drops layer l iff
// u < thr_l = floor(p 2^32).
// Sub-layer granularity (Model Granularity subsection): the attention mask
// takes word 0 and the FFN mask word 1 of the same draw; their tables follow
// each other ([2][L][B], counts [2][L]).
//
// Per token (finer than per sequence; the Tensor Granularity subsection
// leaves it to future work, so the draw is this library's reading): token
// (b, s) drops layer l iff word 2 (FFN mask with sub-layer granularity:
// word 3) of Philox4x32-10 at counter (g, l, t lo, t hi) is below thr_l,
// g = ((b_offset + b) S + s) mod 2^32 its global index.  The kept tokens are
// listed by their rows b S + s in ascending order (so each sequence's kept
// tokens are consecutive) with per-sequence segment offsets.
#include "ld_internal.cuh"

namespace ldk {

// Philox4x32-10 round function and key schedule, from the SC'11 paper:
// multipliers 0xD2511F53 / 0xCD9E8D57, Weyl increments 0x9E3779B9 /
// 0xBB67AE85, ten rounds.
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint2 k) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    if (r > 0) {
      k.x += 0x9E3779B9u;
      k.y += 0xBB67AE85u;
    }
    const uint32_t lo0 = 0xD2511F53u * c.x, hi0 = __umulhi(0xD2511F53u, c.x);
    const uint32_t lo1 = 0xCD9E8D57u * c.z, hi1 = __umulhi(0xCD9E8D57u, c.z);
    c = make_uint4(hi1 ^ c.y ^ k.x, lo1, hi0 ^ c.w ^ k.y, lo0);
  }
  return c;
}

__global__ void mask_compact_kernel(const MaskParams P, unsigned char* __restrict__ mask,
                                    int* __restrict__ kept_idx, int* __restrict__ kept_cnt) {
  __shared__ int warp_off[32];
  __shared__ int base;
  const int w = blockIdx.x / P.L, l = blockIdx.x % P.L;  // mask w of layer l
  const int lane = threadIdx.x & 31, wp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  const unsigned long long thr = P.thr[l];
  const uint2 key = make_uint2((uint32_t)P.seed, (uint32_t)(P.seed >> 32));
  const uint32_t t_lo = (uint32_t)(unsigned long long)P.step, t_hi = (uint32_t)((unsigned long long)P.step >> 32);
  if (threadIdx.x == 0) base = 0;
  __syncthreads();
  for (int b0 = 0; b0 < P.B; b0 += blockDim.x) {
    const int b = b0 + threadIdx.x;
    int keep = 0;
    if (b < P.B) {
      const uint32_t bb = P.granularity == LD_PER_BATCH   ? 0u
                          : P.granularity == LD_PER_SHARD ? (uint32_t)P.b_offset
                                                          : (uint32_t)(P.b_offset + b);
      const uint4 r = philox4x32_10(make_uint4(bb, (uint32_t)l, t_lo, t_hi), key);
      const uint32_t u = w == 0 ? r.x : r.y;
      keep = (unsigned long long)u >= thr;
      mask[(size_t)blockIdx.x * P.B + b] = (unsigned char)keep;
    }
    const unsigned bal = __ballot_sync(0xffffffffu, keep);
    if (lane == 0) warp_off[wp] = __popc(bal);
    __syncthreads();
    if (wp == 0) {
      // exclusive scan of the per-warp counts
      int v = lane < nw ? warp_off[lane] : 0;
      int incl = v;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int n = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += n;
      }
      if (lane < nw) warp_off[lane] = incl - v;
      if (lane == 31) warp_off[31] = incl;  // chunk total (nw <= 31 slots used above)
    }
    __syncthreads();
    if (keep) kept_idx[(size_t)blockIdx.x * P.B + base + warp_off[wp] + __popc(bal & ((1u << lane) - 1u))] = b;
    __syncthreads();
    if (threadIdx.x == 0) base += warp_off[31];
    __syncthreads();
  }
  for (int i = base + threadIdx.x; i < P.B; i += blockDim.x) kept_idx[(size_t)blockIdx.x * P.B + i] = -1;
  if (threadIdx.x == 0) kept_cnt[blockIdx.x] = base;
}

// Per-token masks and kept lists: one block per (mask w, layer l) walks the
// B*S tokens in chunks of blockDim; the exclusive prefix count of the kept
// tokens gives each kept token its compact row and each sequence (its token
// s = 0) its segment start.
__global__ void token_mask_compact_kernel(const MaskParams P, unsigned char* __restrict__ mask,
                                          int* __restrict__ kept_idx, int* __restrict__ kept_cnt,
                                          int* __restrict__ seg) {
  __shared__ int warp_off[32];
  __shared__ int base;
  const int w = blockIdx.x / P.L, l = blockIdx.x % P.L;
  const int lane = threadIdx.x & 31, wp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  const long long T = (long long)P.B * P.S;
  const unsigned long long thr = P.thr[l];
  const uint2 key = make_uint2((uint32_t)P.seed, (uint32_t)(P.seed >> 32));
  const uint32_t t_lo = (uint32_t)(unsigned long long)P.step, t_hi = (uint32_t)((unsigned long long)P.step >> 32);
  const uint32_t g0 = (uint32_t)((unsigned long long)P.b_offset * (unsigned long long)P.S);
  unsigned char* mk = mask + (size_t)blockIdx.x * T;
  int* ki = kept_idx + (size_t)blockIdx.x * T;
  int* sg = seg + (size_t)blockIdx.x * (P.B + 1);
  if (threadIdx.x == 0) base = 0;
  __syncthreads();
  for (long long t0 = 0; t0 < T; t0 += blockDim.x) {
    const long long t = t0 + threadIdx.x;
    int keep = 0;
    if (t < T) {
      const uint4 r = philox4x32_10(make_uint4(g0 + (uint32_t)t, (uint32_t)l, t_lo, t_hi), key);
      const uint32_t u = w == 0 ? r.z : r.w;
      keep = (unsigned long long)u >= thr;
      mk[t] = (unsigned char)keep;
    }
    const unsigned bal = __ballot_sync(0xffffffffu, keep);
    if (lane == 0) warp_off[wp] = __popc(bal);
    __syncthreads();
    if (wp == 0) {
      int v = lane < nw ? warp_off[lane] : 0;
      int incl = v;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int n = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += n;
      }
      if (lane < nw) warp_off[lane] = incl - v;
      if (lane == 31) warp_off[31] = incl;
    }
    __syncthreads();
    const int at = base + warp_off[wp] + __popc(bal & ((1u << lane) - 1u));  // kept tokens before t
    if (t < T && t % P.S == 0) sg[t / P.S] = at;
    if (keep) ki[at] = (int)t;
    __syncthreads();
    if (threadIdx.x == 0) base += warp_off[31];
    __syncthreads();
  }
  for (long long i = base + threadIdx.x; i < T; i += blockDim.x) ki[i] = -1;
  if (threadIdx.x == 0) {
    sg[P.B] = base;
    kept_cnt[blockIdx.x] = (int)(((long long)base + 63) / 64 * 64);  // B*S is a multiple of 64
  }
}

cudaError_t launch_mask_compact(const MaskParams& P, unsigned char* mask, int* kept_idx, int* kept_cnt, int* seg,
                                cudaStream_t st) {
  if (P.granularity == LD_PER_TOKEN) {
    token_mask_compact_kernel<<<P.L * P.nmask, 992, 0, st>>>(P, mask, kept_idx, kept_cnt, seg);
    return cudaGetLastError();
  }
  // at most 31 warps so that slot 31 of warp_off can hold the chunk total
  int threads = ((P.B + 31) / 32) * 32;
  if (threads > 992) threads = 992;
  mask_compact_kernel<<<P.L * P.nmask, threads, 0, st>>>(P, mask, kept_idx, kept_cnt);
  return cudaGetLastError();
}

}  // namespace ldk
