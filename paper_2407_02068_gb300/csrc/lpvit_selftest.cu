// Self-test of the bounded device wait (mbar_wait) that every role of the GEMM uses. One thread
// waits on an mbarrier that nothing arrives on; the wait gives up after its limit, or earlier when
// a second thread raises the CTA's abort flag, and the timeout is recorded in the workspace error
// word exactly as a timed-out GEMM wait records it (read back and cleared by lpvit_check). No copy,
// MMA or TMEM allocation is in flight, so the kernel ends cleanly and the context stays usable.
#include <cstdint>
#include <cuda_runtime.h>

#include "lpvit.h"
#include "lpvit_device.cuh"

namespace lpvit {

constexpr uint64_t SELFTEST_MAX_NS = 10000000000ull;  // 10 s
constexpr unsigned int ERR_SELFTEST_WAIT = 1u << 10;   // a bit the GEMM error bits leave free

__global__ void wait_selftest_kernel(Control *ctl, uint64_t limit_ns, uint64_t abort_after_ns) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(smem_u32(&bar), 1);
    abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  const uint64_t t0 = globaltimer_ns();
  if (threadIdx.x == 0) {
    // phase 0 of a fresh barrier completes only after one arrival, and none comes
    if (!mbar_wait(smem_u32(&bar), 0, &abort_flag, limit_ns)) {
      const uint64_t waited_us = (globaltimer_ns() - t0) / 1000;
      ctl->err_detail = waited_us > 0xffffffffull ? 0xffffffffu : (unsigned int)waited_us;
      __threadfence();
      atomicOr(&ctl->err, ERR_SELFTEST_WAIT);
    }
  } else if (threadIdx.x == 32 && abort_after_ns > 0) {
    // another role of the CTA gives up: raise the abort flag after abort_after_ns (bounded sleep loop)
    while (globaltimer_ns() - t0 < abort_after_ns) __nanosleep(1000);
    *reinterpret_cast<volatile int *>(&abort_flag) = 1;
  }
}

}  // namespace lpvit

using namespace lpvit;

extern "C" lpvit_status lpvit_selftest_wait(void *workspace, uint64_t limit_ns, uint64_t abort_after_ns,
                                            void *stream) {
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) % 256) != 0) return LPVIT_ERR_INVALID_ARG;
  if (limit_ns == 0 || limit_ns > SELFTEST_MAX_NS || abort_after_ns >= limit_ns) return LPVIT_ERR_INVALID_ARG;
  wait_selftest_kernel<<<1, 64, 0, static_cast<cudaStream_t>(stream)>>>(static_cast<Control *>(workspace), limit_ns,
                                                                        abort_after_ns);
  return cudaGetLastError() == cudaSuccess ? LPVIT_OK : LPVIT_ERR_CUDA;
}
