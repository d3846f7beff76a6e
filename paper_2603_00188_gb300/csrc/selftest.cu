// The library's failure path, run on purpose: one CTA waits on an mbarrier
// that nothing arrives on, through the same bounded wait (mbar_wait) every
// tensor-core kernel uses, with a caller-chosen short limit.  The wait gives
// up, records kErrTimeout in the error word and the kernel returns, so the
// host reads STLITE_ETIMEOUT through stlite_device_status and the context
// stays usable.  Nothing faults and nothing hangs.
#include "../../include/stlite.h"
#include "kernels.cuh"
#include "ptx.cuh"

namespace stl {

__global__ void k_wait_selftest(uint32_t* err, unsigned long long limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ uint32_t abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(smem_u32(&bar), 1);
    abort_flag = 0u;
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) mbar_wait(smem_u32(&bar), 0u, err, &abort_flag, limit_ns);  // nothing arrives
  __syncthreads();
}

}  // namespace stl

extern "C" stlite_status stlite_selftest_wait_timeout(void* ws, int64_t limit_ns, void* stream) {
  if (!ws || (reinterpret_cast<uintptr_t>(ws) & 15u) != 0) return STLITE_EINVAL;
  if (limit_ns < 1000 || limit_ns > 2000000000LL) return STLITE_EINVAL;
  stl::k_wait_selftest<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(static_cast<uint32_t*>(ws),
                                                                         (unsigned long long)limit_ns);
  return cudaGetLastError() == cudaSuccess ? STLITE_OK : STLITE_ECUDA;
}
