// lpvit_bsr_linear_noalloc: the block-sparse linear with its scratch memory held by the library.
//
// Who needs it: callers that cannot call cudaMalloc (or any allocator) at the point where they
// run the layer, e.g. code that owns no device allocator because another runtime manages all
// device memory, code recorded while a stream is being captured, or latency-critical paths that
// must not take the allocator's implicit synchronisation. They still pass inputs and outputs; the
// library supplies the workspace.
//
// The workspace lives in one file-scope __device__ array of LPVIT_NOALLOC_SCRATCH_BYTES. Every
// GPU that loads the library holds this array until the process exits. Host code never uses the
// array's symbol as an address: its device address is looked up once per device with
// cudaGetSymbolAddress (with that device current) and cached.
#include <cstdint>
#include <mutex>
#include <cuda_runtime.h>

#include "lpvit.h"
#include "lpvit_device.cuh"

static __device__ __align__(256) unsigned char g_noalloc_scratch[LPVIT_NOALLOC_SCRATCH_BYTES];

namespace {

std::mutex g_noalloc_mu;
void *g_noalloc_ptr[64] = {nullptr};

// Device address of the scratch array for the current device (looked up on first use).
lpvit_status noalloc_scratch(void **out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return LPVIT_ERR_CUDA;
  std::lock_guard<std::mutex> lk(g_noalloc_mu);
  if (!g_noalloc_ptr[dev]) {
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) return LPVIT_ERR_CUDA;
    g_noalloc_ptr[dev] = p;
  }
  *out = g_noalloc_ptr[dev];
  return LPVIT_OK;
}

}  // namespace

extern "C" lpvit_status lpvit_bsr_linear_noalloc(const lpvit_bsr *bsr, const void *X, int64_t m, int64_t ldx,
                                                 const float *bias, void *Y, int64_t ldy, lpvit_dtype y_dtype,
                                                 int gelu, void *stream) {
  if (!bsr || m < 0) return LPVIT_ERR_INVALID_ARG;
  if (m == 0) return LPVIT_OK;
  const size_t need = lpvit_workspace_bytes(bsr, m);
  if (need == 0) return LPVIT_ERR_INVALID_ARG;
  if (need > (size_t)LPVIT_NOALLOC_SCRATCH_BYTES) return LPVIT_ERR_WORKSPACE;
  void *ws = nullptr;
  const lpvit_status st = noalloc_scratch(&ws);
  if (st != LPVIT_OK) return st;
  // The array keeps whatever the previous call left; the work-queue counters and the error word
  // at its start must begin at zero (partial sums are always written before they are read), so
  // clear them on the caller's stream.
  size_t clear = sizeof(lpvit::Control);
  if (clear > need) clear = need;
  if (cudaMemsetAsync(ws, 0, clear, static_cast<cudaStream_t>(stream)) != cudaSuccess) return LPVIT_ERR_CUDA;
  return gelu ? lpvit_bsr_linear_gelu(bsr, X, m, ldx, bias, Y, ldy, y_dtype, ws, LPVIT_NOALLOC_SCRATCH_BYTES, stream)
              : lpvit_bsr_linear(bsr, X, m, ldx, bias, Y, ldy, y_dtype, ws, LPVIT_NOALLOC_SCRATCH_BYTES, stream);
}
