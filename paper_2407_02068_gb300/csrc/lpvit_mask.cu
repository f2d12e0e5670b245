// Block mask from first-order Taylor scores (Sec. 3.1, block-structured pruning within a layer):
// the neuron score |W . grad W|, a 2D average pooling with the block (bn rows by bk columns) as
// window and stride, and the bottom-ranked blocks eliminated at the layer's pruning ratio.
//
// score kernel (one thread per block, grid-stride): the block's |w * g| summed in double in
//   row-major order, then divided by bn * bk. The product of a bf16 weight and a float32 gradient is
//   exact in double, so the sum is the same sequence of correctly rounded additions as a plain
//   sequential loop: the scores are bit-identical to any such loop.
// select kernel (one thread per block, scores streamed through shared memory in tiles): block t is
//   kept when fewer than `keep` blocks rank ahead of it, where u ranks ahead of t if its score is
//   higher, or equal with a lower linear block index.
#include <cmath>
#include <cstdint>
#include <cuda_runtime.h>

#include "lpvit.h"

namespace lpvit {

namespace {

constexpr int MASK_THREADS = 256;
constexpr int SELECT_TILE = 2048;          // scores per shared-memory tile (16 KB)
constexpr int64_t MAX_MASK_BLOCKS = 1 << 20;

template <int BK>
__global__ void __launch_bounds__(MASK_THREADS)
score_kernel(const uint16_t *__restrict__ W, const float *__restrict__ G, int n, int k, int bn,
             double *__restrict__ scores) {
  const int np = n / bn, kb = k / BK;
  const int64_t total = (int64_t)np * kb;
  for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total; t += (int64_t)gridDim.x * blockDim.x) {
    const int r = (int)(t / kb), j = (int)(t - (int64_t)r * kb);
    double sum = 0.0;
    for (int i = 0; i < bn; ++i) {
      const int64_t e0 = (int64_t)(r * bn + i) * k + (int64_t)j * BK;
      // the row's BK weights and BK gradients as 16-byte vectors, then the sequential sum
      uint4 wv[BK / 8];
      float4 gv[BK / 4];
#pragma unroll
      for (int v = 0; v < BK / 8; ++v) wv[v] = __ldg(reinterpret_cast<const uint4 *>(W + e0) + v);
#pragma unroll
      for (int v = 0; v < BK / 4; ++v) gv[v] = __ldg(reinterpret_cast<const float4 *>(G + e0) + v);
      const uint16_t *wh = reinterpret_cast<const uint16_t *>(wv);
      const float *gf = reinterpret_cast<const float *>(gv);
#pragma unroll
      for (int l = 0; l < BK; ++l) {
        const double w = (double)__uint_as_float((uint32_t)wh[l] << 16);
        sum += fabs(w * (double)gf[l]);
      }
    }
    scores[t] = sum / ((double)bn * (double)BK);
  }
}

__global__ void __launch_bounds__(MASK_THREADS)
select_kernel(const double *__restrict__ scores, int64_t total, int64_t keep, uint8_t *__restrict__ mask) {
  __shared__ double tile[SELECT_TILE];
  const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const double st = t < total ? scores[t] : 0.0;
  int64_t ahead = 0;
  for (int64_t base = 0; base < total; base += SELECT_TILE) {
    const int len = total - base < SELECT_TILE ? (int)(total - base) : SELECT_TILE;
    __syncthreads();
    for (int i = threadIdx.x; i < len; i += blockDim.x) tile[i] = scores[base + i];
    __syncthreads();
    if (t < total) {
      for (int i = 0; i < len; ++i) {
        const double su = tile[i];
        const int64_t u = base + i;
        ahead += (su > st || (su == st && u < t)) ? 1 : 0;
      }
    }
  }
  if (t < total) mask[t] = ahead < keep ? 1 : 0;
}

bool aligned_to(const void *p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

}  // namespace
}  // namespace lpvit

using namespace lpvit;

extern "C" lpvit_status lpvit_taylor_block_mask(const void *W, const float *G, int32_t n, int32_t k, int32_t bn,
                                                int32_t bk, double prune_ratio, double *scores, uint8_t *mask,
                                                void *stream) {
  if ((bn != 16 && bn != 32 && bn != 64) || (bk != 16 && bk != 32 && bk != 64)) return LPVIT_ERR_UNSUPPORTED;
  if (n <= 0 || k <= 0 || n > 65536 || k > 65536 || n % bn || k % bk) return LPVIT_ERR_INVALID_ARG;
  if (!(prune_ratio >= 0.0 && prune_ratio <= 1.0)) return LPVIT_ERR_INVALID_ARG;  // also rejects NaN
  if (!W || !G || !scores || !mask) return LPVIT_ERR_INVALID_ARG;
  if (!aligned_to(W, 16) || !aligned_to(G, 16) || !aligned_to(scores, 8)) return LPVIT_ERR_INVALID_ARG;
  const int64_t total = (int64_t)(n / bn) * (k / bk);
  if (total > MAX_MASK_BLOCKS) return LPVIT_ERR_UNSUPPORTED;
  // eliminated = round(alpha * blocks), half away from zero; the rest are kept
  const int64_t pruned = (int64_t)floor(prune_ratio * (double)total + 0.5);
  const int64_t keep = total - pruned;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int grid = (int)((total + MASK_THREADS - 1) / MASK_THREADS);
  const uint16_t *Wh = static_cast<const uint16_t *>(W);
  switch (bk) {
    case 16: score_kernel<16><<<grid, MASK_THREADS, 0, s>>>(Wh, G, n, k, bn, scores); break;
    case 32: score_kernel<32><<<grid, MASK_THREADS, 0, s>>>(Wh, G, n, k, bn, scores); break;
    default: score_kernel<64><<<grid, MASK_THREADS, 0, s>>>(Wh, G, n, k, bn, scores); break;
  }
  if (cudaGetLastError() != cudaSuccess) return LPVIT_ERR_CUDA;
  select_kernel<<<grid, MASK_THREADS, 0, s>>>(scores, total, keep, mask);
  return cudaGetLastError() == cudaSuccess ? LPVIT_OK : LPVIT_ERR_CUDA;
}
