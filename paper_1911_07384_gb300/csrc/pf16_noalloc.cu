// Weight gradient for callers that cannot hand the library any scratch memory.
//
// pf16_conv_wgrad needs a caller-provided workspace for its split-K FP16
// partial sums.  Some callers have no way to provide one: a host framework
// that plans every byte of device memory itself and does not let plug-ins ask
// for more, a deployment that forbids device allocation once set-up is over,
// or a thin binding from a language with no CUDA allocator at hand.  A
// cudaMalloc in the middle of a training loop is also unwelcome because it can
// stall the whole device.  For them, pf16_conv_wgrad_noalloc keeps its
// scratch in one fixed array compiled into the library, so it allocates
// nothing at call time.
//
// The array is PF16_WGRAD_NOALLOC_SCRATCH_BYTES (32 MiB) per device, about the size of
// the default cuBLAS workspace on recent GPUs; every device that loads this
// part of the library keeps it until the process exits.  All calls share it.
#include <cuda_runtime.h>

#include <cstdint>
#include <mutex>

#include "../../include/pf16.h"

namespace {

constexpr size_t kPf16NoallocScratchBytes = PF16_WGRAD_NOALLOC_SCRATCH_BYTES;

// The shared scratch.  Split-K partial sums of the weight gradient live here
// between the GEMM and its reduction within one call; every element a call
// reads was written earlier in the same call, so nothing needs clearing.
static __device__ __align__(256) uint16_t g_pf16_noalloc_scratch[kPf16NoallocScratchBytes / 2];

constexpr int kMaxDev = 64;
std::mutex g_mu;
void* g_scratch_addr[kMaxDev] = {nullptr};

// Device address of the scratch array on the current device (resolved once per
// device, with that device current).  In host code the array's name is only a
// host-side stand-in, so kernels must be given this address instead.
int scratch_address(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDev) return PF16_ERR_CUDA;
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_scratch_addr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_pf16_noalloc_scratch) != cudaSuccess || p == nullptr)
      return PF16_ERR_CUDA;
    g_scratch_addr[dev] = p;
  }
  *out = g_scratch_addr[dev];
  return PF16_OK;
}

}  // namespace

extern "C" int pf16_conv_wgrad_noalloc(const pf16_conv_desc* d, const uint16_t* x, const uint16_t* dy,
                                       uint16_t* dw, uint32_t flags, void* stream) {
  if (!d) return PF16_ERR_NULL;
  const size_t need = pf16_conv_workspace_size(d, PF16_PASS_WGRAD);
  if (need > kPf16NoallocScratchBytes) return PF16_ERR_WORKSPACE;
  void* scratch = nullptr;
  const int rc = scratch_address(&scratch);
  if (rc != PF16_OK) return rc;
  return pf16_conv_wgrad(d, x, dy, dw, scratch, kPf16NoallocScratchBytes, flags, stream);
}
