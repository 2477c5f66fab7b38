// Self-test of the bounded device waits used by the FFN kernels.
//
// A kernel waits on an mbarrier that nothing ever arrives at, through the
// same bounded wait (mbar_wait) that every pipeline wait of the library
// uses.  The wait must give up after its time budget, the kernel must report
// XS_DEV_TIMEOUT in the caller's xs_stats and return, and the CUDA context
// must stay usable.  No fault, trap or unbounded loop is involved.
#include <cuda_runtime.h>

#include "tc_ptx.cuh"
#include "xs_internal.cuh"

namespace xs {
namespace {

__global__ void wait_timeout_kernel(xs_stats *stats, unsigned long long budget_ns) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    ptx::mbar_init(ptx::smem_u32(&bar), 1);
    abort_flag = 0;
    ptx::fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    const uint64_t t0 = ptx::globaltimer();
    const bool ok = ptx::mbar_wait(ptx::smem_u32(&bar), 0, budget_ns, &abort_flag);
    const uint64_t waited = ptx::globaltimer() - t0;
    stats->status = ok ? XS_DEV_OK : XS_DEV_TIMEOUT;
    stats->reserved[0] = static_cast<int32_t>(waited / 1000000ull);  // milliseconds waited
    // Complete the barrier's phase so that nothing is left pending.
    ptx::mbar_arrive(ptx::smem_u32(&bar));
  }
}

}  // namespace
}  // namespace xs

extern "C" int xshare_selftest_wait_timeout(xs_stats *stats, uint64_t budget_ns,
                                            xs_stream_t stream) {
  if (stats == nullptr) return XS_ERR_NULL;
  if (budget_ns == 0 || budget_ns > 2000000000ull) return XS_ERR_PARAM;
  xs::wait_timeout_kernel<<<1, 32, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
      stats, static_cast<unsigned long long>(budget_ns));
  return cudaGetLastError() == cudaSuccess ? XS_OK : XS_ERR_CUDA;
}
