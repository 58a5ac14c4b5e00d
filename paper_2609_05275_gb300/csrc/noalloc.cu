// ld_rmsnorm_backward_noalloc: the RMSNorm-backward step of ld_rmsnorm_backward
// for callers that cannot allocate device memory.
//
// Some callers cannot call cudaMalloc (or any allocating routine) at the
// point where they need this step: code recorded into a CUDA graph with a
// global capture mode, where allocation calls are refused while the stream is
// capturing; runtimes whose device memory is all owned by another allocator
// that this library cannot reach; latency-critical paths that must not enter
// an allocator at all.  For them the per-block partial sums of the gain
// gradient live in a fixed array in this file instead of a caller buffer.
//
// The array is a file-scope __device__ object, so every GPU that loads the
// library holds it (kNoallocScratchFloats floats = 10 MiB) until the process
// exits.  Host code cannot use the array's name as a device address: on the
// first call on each device (with that device current) the entry point asks
// the runtime for the address with cudaGetSymbolAddress and keeps it, keyed
// by the device and its current context.  That first call should therefore
// come before any stream capture.  After cudaDeviceReset the device has a new
// primary context in which the module, and so the array, is loaded afresh:
// the next call sees the new context and looks the address up again (that
// call, too, should come before any capture).
//
// All calls share the one array.  Every call writes each partial sum it later
// reads (block b fills row b completely before the column sum runs), so
// nothing has to start at zero; but calls that overlap on the GPU (two
// streams, or two host threads) race on the array and must be serialised by
// the caller.
#include <cuda.h>

#include <mutex>

#include "ld_internal.cuh"

namespace {

constexpr long long kNoallocScratchFloats = 2621440;  // 10 MiB
constexpr int kMaxDevices = 64;

__device__ __align__(256) float g_noalloc_scratch[kNoallocScratchFloats];

struct ScratchAddr {
  CUcontext ctx;  // the context the address belongs to
  float* ptr;
};
ScratchAddr g_scratch_addr[kMaxDevices] = {};
std::mutex g_scratch_mu;

// The driver's cuCtxGetCurrent, reached through the runtime (the library
// links the runtime only).
using CtxGetCurrentFn = CUresult (*)(CUcontext*);
CtxGetCurrentFn ctx_get_current() {
  static const CtxGetCurrentFn fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      return static_cast<CtxGetCurrentFn>(nullptr);
    return reinterpret_cast<CtxGetCurrentFn>(p);
  }();
  return fn;
}

// Device address of g_noalloc_scratch on the current device, looked up once
// per (device, context); null on failure.
float* scratch_address() {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  CtxGetCurrentFn get = ctx_get_current();
  CUcontext ctx = nullptr;
  if (!get || get(&ctx) != CUDA_SUCCESS) return nullptr;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  ScratchAddr& a = g_scratch_addr[dev];
  if (!ctx || !a.ptr || a.ctx != ctx) {
    // the lookup also makes the device's primary context current when no
    // context is yet
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return nullptr;
    if (get(&ctx) != CUDA_SUCCESS || !ctx) return nullptr;
    a.ctx = ctx;
    a.ptr = static_cast<float*>(p);
  }
  return a.ptr;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

}  // namespace

extern "C" ld_status ld_rmsnorm_backward_noalloc(int B, int S, int d, const float* dyn, const void* xs,
                                                 const float* rstd, const void* gamma, const int* kept_idx,
                                                 const int* kept_cnt, float* dx, void* next, float scale,
                                                 float* dgamma, void* stream) {
  if (B < 1 || S < 1 || d < 8 || d % 8 || d > 16384 || (long long)B * S > (1ll << 30)) return LD_ERR_SHAPE;
  const void* ps[] = {dyn, xs, rstd, gamma, dx, dgamma};
  for (const void* p : ps)
    if (!p || !aligned16(p)) return LD_ERR_ARG;
  if (!kept_idx || !kept_cnt || (next && !aligned16(next))) return LD_ERR_ARG;
  long long nb = ((long long)B * S + 7) / 8;
  if (nb > 320) nb = 320;
  if (nb * d > kNoallocScratchFloats) return LD_ERR_SHAPE;  // partial sums would not fit the fixed array
  float* scratch = scratch_address();
  if (!scratch) return LD_ERR_CUDA;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (ldk::launch_rmsnorm_bwd<ldk::bf16>(dyn, static_cast<const float*>(xs), rstd,
                                         static_cast<const ldk::bf16*>(gamma), dx, kept_idx, kept_cnt, S, d, B * S,
                                         scale, static_cast<ldk::bf16*>(next), scratch, (int)nb, st) != cudaSuccess)
    return LD_ERR_CUDA;
  if (ldk::launch_colsum(scratch, (int)nb, d, dgamma, st) != cudaSuccess) return LD_ERR_CUDA;
  return LD_OK;
}
