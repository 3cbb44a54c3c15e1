// mcpu_selftest_wait_timeout: a check of the give-up path of the bounded
// mbarrier waits, runnable on a GPU without a fault or a hang.
//
// Every wait in the attention kernels is bounded by kWaitTimeoutNs of
// %globaltimer and, when it runs out, ORs kStatusTimeout into the workspace
// status word and lets the kernel return. Valid or invalid inputs cannot make
// one of those waits run out (a page outside the pool becomes a zero-filled
// copy, not a missing one), so this kernel builds the situation directly: a
// shared-memory mbarrier that nothing ever arrives at, waited on by a whole
// warp with the same mbar_wait the decode kernels use, exactly as they use it
// (every lane polls, the warp votes). Beside it a second warp waits on a
// barrier whose phase does complete, which must return at once.
#include "../../include/mcpu.h"
#include "common.cuh"

namespace {

using namespace mcpu;

// One CTA of 64 threads. report[0]: the completing wait's result (1),
// report[1]: the never-completing wait's result (0), report[2]: how long
// that wait took in ns, report[3]: the library's wait limit in ns.
__global__ void selftest_wait_kernel(int32_t* status_word, int64_t* report) {
  __shared__ __align__(8) uint64_t bars[2];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    mbar_init(smem_addr(&bars[0]), 1);  // nothing arrives here
    mbar_init(smem_addr(&bars[1]), 1);  // one arrival completes phase 0
    fence_barrier_init();
  }
  __syncthreads();
  if (warp == 0) {
    const uint64_t t0 = global_timer_ns();
    const bool ok = __any_sync(0xffffffffu, mbar_wait(smem_addr(&bars[0]), 0));
    const uint64_t t1 = global_timer_ns();
    if (lane == 0) {
      if (!ok) atomicOr(status_word, kStatusTimeout);
      report[1] = ok ? 1 : 0;
      report[2] = (int64_t)(t1 - t0);
      report[3] = (int64_t)kWaitTimeoutNs;
    }
  } else {
    if (lane == 0) mbar_arrive(smem_addr(&bars[1]));
    __syncwarp();
    const bool ok = __any_sync(0xffffffffu, mbar_wait(smem_addr(&bars[1]), 0));
    if (lane == 0) report[0] = ok ? 1 : 0;
  }
}

}  // namespace

extern "C" mcpu_status mcpu_selftest_wait_timeout(void* workspace, int64_t* report, mcpu_stream_t stream) {
  if (workspace == nullptr || report == nullptr) return MCPU_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(workspace) % 4 != 0 || reinterpret_cast<uintptr_t>(report) % 8 != 0)
    return MCPU_ERR_INVALID_ARG;
  selftest_wait_kernel<<<1, 64, 0, reinterpret_cast<cudaStream_t>(stream)>>>(static_cast<int32_t*>(workspace),
                                                                             report);
  return cudaGetLastError() == cudaSuccess ? MCPU_OK : MCPU_ERR_CUDA;
}
