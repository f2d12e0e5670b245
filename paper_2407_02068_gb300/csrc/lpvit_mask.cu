// Block mask from first-order Taylor scores (Sec. 3.1, block-structured pruning within a layer):
// the neuron score |W . grad W|, a 2D average pooling with the block (bn rows by bk columns) as
// window and stride, and the bottom-ranked blocks eliminated at the layer's pruning ratio.
//
// score kernel (one warp per block, grid-stride; lane i sums rows i and i + 32, lane 0 then adds
//   the row sums in row order): in float32, the gradient's precision, each
//   product |w * g| rounded to float, each block row summed in order, the row sums summed in row
//   order; the total widened to double and divided by bn * bk. Every step is one IEEE operation in
//   a fixed order, so the scores are bit-identical to a plain loop doing the same operations. (The
//   double pipe of this GPU retires one warp instruction per 64 cycles per SM; the float path
//   keeps a block's few thousand products off it.)
// select kernel (one thread per block, scores streamed through shared memory in tiles): block t is
//   kept when fewer than `keep` blocks rank ahead of it, where u ranks ahead of t if its score is
//   higher, or equal with a lower linear block index. Scores are sums of magnitudes (>= +0, finite),
//   and for such doubles the IEEE bit patterns read as unsigned integers order exactly as the
//   values, so the comparisons run on 64-bit integer keys (the FP64 pipe is narrow on this GPU).
//   A CTA of SELECT_WARPS warps ranks 32 blocks (one per lane); the keys stream through shared
//   memory in tiles and each warp compares its lanes' blocks with its share of every tile; the
//   warps' counts are then added.
// The score kernel runs warps in CTAs of MASK_CTA threads so that a few thousand blocks still
//   spread over every SM.
#include <cmath>
#include <cstdint>
#include <cuda_runtime.h>

#include "lpvit.h"
#include "lpvit_taylor.h"

namespace lpvit {

namespace {

constexpr int MASK_THREADS = 256;          // upper bound of MASK_CTA (launch bounds)
constexpr int MASK_CTA = 128;              // threads per CTA of the score launch (4 blocks)
constexpr int SELECT_TILE = 2048;          // keys per shared-memory tile (16 KB)
constexpr int SELECT_WARPS = 8;
constexpr int64_t MAX_MASK_BLOCKS = 1 << 20;

// The float32 sum of |w * g| over row i of block (r, j), in column order.
template <int BK>
__device__ __forceinline__ float row_sum(const uint16_t *__restrict__ W, const float *__restrict__ G, int64_t e0) {
  uint4 wv[BK / 8];
  float4 gv[BK / 4];
#pragma unroll
  for (int v = 0; v < BK / 8; ++v) wv[v] = __ldg(reinterpret_cast<const uint4 *>(W + e0) + v);
#pragma unroll
  for (int v = 0; v < BK / 4; ++v) gv[v] = __ldg(reinterpret_cast<const float4 *>(G + e0) + v);
  const uint16_t *wh = reinterpret_cast<const uint16_t *>(wv);
  const float *gf = reinterpret_cast<const float *>(gv);
  float row = 0.f;
#pragma unroll
  for (int l = 0; l < BK; ++l) row = __fadd_rn(row, fabsf(__fmul_rn(__uint_as_float((uint32_t)wh[l] << 16), gf[l])));
  return row;
}

template <int BK>
__global__ void __launch_bounds__(MASK_THREADS)
score_kernel(const uint16_t *__restrict__ W, const float *__restrict__ G, int n, int k, int bn,
             double *__restrict__ scores) {
  const int np = n / bn, kb = k / BK;
  const int lane = threadIdx.x & 31;
  const int64_t total = (int64_t)np * kb;
  const int64_t warps = (int64_t)gridDim.x * (blockDim.x / 32);
  for (int64_t t = (int64_t)blockIdx.x * (blockDim.x / 32) + (threadIdx.x >> 5); t < total; t += warps) {
    const int r = (int)(t / kb), j = (int)(t - (int64_t)r * kb);
    float lo = 0.f, hi = 0.f;  // rows lane and lane + 32
    if (lane < bn) lo = row_sum<BK>(W, G, (int64_t)(r * bn + lane) * k + (int64_t)j * BK);
    if (lane + 32 < bn) hi = row_sum<BK>(W, G, (int64_t)(r * bn + lane + 32) * k + (int64_t)j * BK);
    float sum = 0.f;
    for (int i = 0; i < bn; ++i) {
      const float v = __shfl_sync(0xffffffffu, i < 32 ? lo : hi, i & 31);
      sum = __fadd_rn(sum, v);
    }
    if (lane == 0) scores[t] = (double)sum / ((double)bn * (double)BK);
  }
}

// mask (if not null): 1 for the `keep` best-ranked blocks; rank (if not null): the number of blocks
// ranked ahead of each block (0 = the best).
__global__ void __launch_bounds__(32 * SELECT_WARPS)
select_kernel(const double *__restrict__ scores, int64_t total, int64_t keep, uint8_t *__restrict__ mask,
              int32_t *__restrict__ rank) {
  __shared__ unsigned long long tile[SELECT_TILE];
  __shared__ long long part[SELECT_WARPS][32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t t = (int64_t)blockIdx.x * 32 + lane;
  const unsigned long long st = t < total ? (unsigned long long)__double_as_longlong(scores[t]) : 0ull;
  long long ahead = 0;
  for (int64_t base = 0; base < total; base += SELECT_TILE) {
    const int len = total - base < SELECT_TILE ? (int)(total - base) : SELECT_TILE;
    __syncthreads();
    for (int i = threadIdx.x; i < len; i += blockDim.x)
      tile[i] = (unsigned long long)__double_as_longlong(scores[base + i]);
    __syncthreads();
    const int lo = (int)((int64_t)len * warp / SELECT_WARPS), hi = (int)((int64_t)len * (warp + 1) / SELECT_WARPS);
    if (t < total) {
      for (int i = lo; i < hi; ++i) {
        const unsigned long long su = tile[i];
        const int64_t u = base + i;
        ahead += (su > st || (su == st && u < t)) ? 1 : 0;
      }
    }
  }
  part[warp][lane] = ahead;
  __syncthreads();
  if (warp == 0 && t < total) {
    long long tot = 0;
#pragma unroll
    for (int w = 0; w < SELECT_WARPS; ++w) tot += part[w][lane];
    if (mask) mask[t] = tot < keep ? 1 : 0;
    if (rank) rank[t] = (int32_t)tot;
  }
}

bool aligned_to(const void *p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

}  // namespace

cudaError_t launch_block_scores(const uint16_t *W, const float *G, int n, int k, int bn, int bk, double *scores,
                                cudaStream_t s) {
  const int64_t total = (int64_t)(n / bn) * (k / bk);
  const int64_t want = (total + MASK_CTA / 32 - 1) / (MASK_CTA / 32);
  const int grid = (int)(want < 152 * 16 ? want : 152 * 16);
  switch (bk) {
    case 16: score_kernel<16><<<grid, MASK_CTA, 0, s>>>(W, G, n, k, bn, scores); break;
    case 32: score_kernel<32><<<grid, MASK_CTA, 0, s>>>(W, G, n, k, bn, scores); break;
    case 64: score_kernel<64><<<grid, MASK_CTA, 0, s>>>(W, G, n, k, bn, scores); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

cudaError_t launch_block_rank(const double *scores, int64_t total, int64_t keep, uint8_t *mask, int32_t *rank,
                              cudaStream_t s) {
  const int grid = (int)((total + 31) / 32);
  select_kernel<<<grid, 32 * SELECT_WARPS, 0, s>>>(scores, total, keep, mask, rank);
  return cudaGetLastError();
}

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
  if (launch_block_scores(static_cast<const uint16_t *>(W), G, n, k, bn, bk, scores, s) != cudaSuccess)
    return LPVIT_ERR_CUDA;
  return launch_block_rank(scores, total, keep, mask, nullptr, s) == cudaSuccess ? LPVIT_OK : LPVIT_ERR_CUDA;
}
