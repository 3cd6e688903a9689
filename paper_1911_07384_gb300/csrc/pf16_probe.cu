// Tensor-core rate probe: the 16-bit dense tcgen05 rate with FP16 (or FP32)
// accumulation, measured by the library's own MMA-only kernel, so that the
// conv rooflines can be read against the rate of the very instruction the
// convolutions issue (kind::f16, M = 128, f16 operands, accumulator in TMEM).
#include <cuda_runtime.h>

#include <cstdint>

#include "pf16_internal.h"
#include "pf16_ptx.cuh"

namespace pf16 {

// One CTA per SM: the dynamic shared memory request keeps a second CTA off the
// SM, so that no CTA's 512-column TMEM allocation waits on another's.
constexpr int kProbeSmem = 200 * 1024;
constexpr int kProbeThreads = 128;

// A (128 x 64) and B (n x 64) K-major 128B-swizzled tiles of zeros; thread 0
// issues reps x 4 MMAs (K = 64 per group) into one accumulator (chains = 1:
// every MMA accumulates onto the previous one, as along a GEMM's K loop) or
// into two in turn (chains = 2), then waits for their completion on an
// mbarrier (bounded; on expiry the status word records PF16_ERR_TIMEOUT and
// the thread waits once more, again bounded, before TMEM is freed).
__global__ void __launch_bounds__(kProbeThreads, 1)
    k_tc_rate(uint32_t idesc, int n, int chains, int reps, int* status, unsigned long long wait_ns) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  __shared__ uint64_t bar;
  __shared__ uint32_t tslot;
  __shared__ int drained;  // the MMAs are known complete: their TMEM may be released
  const int warp = threadIdx.x >> 5;
  const int words = (kBM * 64 * 2 + n * 64 * 2) / 16;
  for (int i = threadIdx.x; i < words; i += blockDim.x)
    st_shared_v4(smem_u32(smem) + (uint32_t)i * 16u, make_uint4(0u, 0u, 0u, 0u));
  fence_proxy_async_smem();  // the operand writes, before the tensor core reads them
  if (threadIdx.x == 0) {
    mbar_init(smem_u32(&bar), 1);
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc(smem_u32(&tslot), 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tslot;
  if (threadIdx.x == 0) {
    const uint64_t a0 = smem_desc(smem_u32(smem), 16, 1024, 2);
    const uint64_t b0 = smem_desc(smem_u32(smem + kBM * 64 * 2), 16, 1024, 2);
#pragma unroll 1
    for (int it = 0; it < reps; ++it) {
      const uint32_t d = tmem + (uint32_t)((chains == 2 ? (it & 1) : 0) * n);
#pragma unroll
      for (int kk = 0; kk < 4; ++kk)  // 32-byte K steps: 2 in the descriptor's 16-byte units
        tc_mma_f16(d, a0 + (uint64_t)(kk * 2), b0 + (uint64_t)(kk * 2), idesc, (it >= chains || kk > 0) ? 1u : 0u);
    }
    tc_commit(smem_u32(&bar));
    drained = 1;
    if (!mbar_wait(smem_u32(&bar), 0, wait_ns)) {
      atomicCAS(status, 0, -7);  // PF16_ERR_TIMEOUT
      // a second bounded wait; if the MMAs still have not completed, their
      // TMEM is left allocated rather than released under them
      drained = mbar_wait(smem_u32(&bar), 0, 1000000000ull) ? 1 : 0;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0 && drained) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

cudaError_t launch_tc_rate(uint32_t idesc, int n, int chains, int reps, int grid, int* status,
                           unsigned long long wait_ns, cudaStream_t s) {
  static bool attr_set[64] = {false};  // per device ordinal
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 64 && !attr_set[dev]) {
    cudaError_t e = cudaFuncSetAttribute(k_tc_rate, cudaFuncAttributeMaxDynamicSharedMemorySize, kProbeSmem);
    if (e != cudaSuccess) return e;
    attr_set[dev] = true;
  }
  k_tc_rate<<<grid, kProbeThreads, kProbeSmem, s>>>(idesc, n, chains, reps, status, wait_ns);
  return counted_launches(1);
}

}  // namespace pf16
