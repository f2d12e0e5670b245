// Layer-wise pruning-ratio allocation (Sec. 3.4, 3.5): the per-layer curve
//   delta(alpha) = g . dW(alpha) + 1/2 dW(alpha)^T H dW(alpha),
// H the empirical Fisher kappa I + (1/N) sum_n g_n g_n^T, dW(alpha) = -W on the blocks that the
// Sec. 3.1 Taylor ranking eliminates at ratio alpha, g the mean of the N per-sample gradients g_n;
// and the lambda search of Eq. langrangian2 over those curves.
//
// The curve follows the incremental update of Eq. update: raising alpha from alpha_{k-1} to
// alpha_k prunes a further set of blocks, d = dW_k - dW_{k-1} (disjoint from dW_{k-1}), and
//   delta_k = delta_{k-1} + g . d + 1/2 d^T H d + dW_{k-1}^T H d.
// With H in its low-rank form and p_n = g_n . dW_{k-1}, q_n = g_n . d:
//   d^T H d = kappa |d|^2 + (1/N) sum q_n^2,   dW_{k-1}^T H d = (1/N) sum p_n q_n,
// so only per-block sums are needed, never a D x D matrix:
//   s[n][t] = sum_{e in t} g_n[e] W[e],  gw[t] = sum g[e] W[e],  w2[t] = sum W[e]^2.
//
// mean_grad_kernel  (grid-stride over the D weights): g[e] = (sum_n g_n[e]) / N in float32, the
//                   sum in sample order (the gradients' own precision; IEEE adds and division).
// block_sums_kernel (one warp per block and sample, plus one per block for gw / w2): lane l adds
//                   the block's elements l, l+32, ... in row-major order, then a fixed shuffle tree.
//                   A bf16 weight times a float32 gradient has at most 32 significant bits, so
//                   each product is taken exactly as a float pair (p = w * g rounded, plus
//                   fma(w, g, -p)), and sums are carried as float pairs with the error-free
//                   two-sum of Knuth (TAOCP vol. 2, 4.2.2): about 48 significant bits at the
//                   float32 rate. (The double pipe of this GPU retires one warp instruction per
//                   64 cycles per SM, the float pipe dozens per cycle.) Results stay float pairs.
// order_kernel      order[rank[t]] = t: the blocks in rank order (the lowest scores last).
// step_sums_kernel  (one warp per step and sample, plus one per step for g . d and |d|^2): the
//                   float-pair sum over the step's newly pruned rank range, lanes striding it, a
//                   fixed shuffle tree, widened to double once.
// increment_kernel  (one warp per step): p_n = sum of the earlier steps' q_n, then
//                   delta_k - delta_{k-1} = lin + (kappa sq + sum q^2 / N) / 2 + sum p q / N.
// prefix_kernel     (one thread): delta_k = sum of the increments up to k, delta_0 = 0.
#include <algorithm>
#include <cmath>
#include <cstdint>
#include <vector>
#include <cuda_runtime.h>

#include "lpvit.h"
#include "lpvit_taylor.h"

namespace lpvit {

namespace {

constexpr int ALLOC_THREADS = 256;
constexpr int MAX_SAMPLES = 1024;
constexpr int MAX_STEPS = 4096;
constexpr int64_t MAX_ALLOC_BLOCKS = 1 << 20;

__global__ void __launch_bounds__(ALLOC_THREADS)
mean_grad_kernel(const float *__restrict__ G, int nsamples, int64_t D, float *__restrict__ g) {
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < D; e += (int64_t)gridDim.x * blockDim.x) {
    float acc = 0.f;
    for (int i = 0; i < nsamples; ++i) acc = __fadd_rn(acc, __ldg(G + (int64_t)i * D + e));
    g[e] = __fdiv_rn(acc, (float)nsamples);
  }
}

// (hi, lo) += x exactly up to the rounding of lo (two-sum: hi + x = t + err exactly).
__device__ __forceinline__ void pair_add(float &hi, float &lo, float x) {
  const float t = __fadd_rn(hi, x);
  const float bp = __fsub_rn(t, hi);
  const float err = __fadd_rn(__fsub_rn(hi, __fsub_rn(t, bp)), __fsub_rn(x, bp));
  hi = t;
  lo = __fadd_rn(lo, err);
}

// (hi, lo) += (bh, bl): two-sum of the high parts, the low parts and the error added.
__device__ __forceinline__ void pair_add2(float &hi, float &lo, float bh, float bl) {
  pair_add(hi, lo, bh);
  lo = __fadd_rn(lo, bl);
}

__device__ __forceinline__ void warp_pair_sum(float &hi, float &lo) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float oh = __shfl_xor_sync(0xffffffffu, hi, o), ol = __shfl_xor_sync(0xffffffffu, lo, o);
    pair_add2(hi, lo, oh, ol);
  }
}

__device__ __forceinline__ double warp_sum(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Warp w handles block t and sample group u (samples [u*SPW, u*SPW + SPW) of N; the last group,
// u == groups - 1, gives gw[t] and w2[t] from g instead). Lane l takes the block's 4-element chunks
// l, l + 32, ... in row-major order (a chunk stays inside one block row: bk is a multiple of 4),
// loading 4 weights and, per sample, 4 gradients as vectors.
constexpr int SPW = 4;  // samples per warp

template <int BK>
__global__ void __launch_bounds__(ALLOC_THREADS)
block_sums_kernel(const uint16_t *__restrict__ W, const float *__restrict__ G, const float *__restrict__ g,
                  int nsamples, int n, int k, int bn, float2 *__restrict__ s, float2 *__restrict__ gw,
                  float2 *__restrict__ w2) {
  const int lane = threadIdx.x & 31;
  constexpr int CPR = BK / 4;  // chunks per block row
  const int kb = k / BK;
  const int64_t T = (int64_t)(n / bn) * kb;
  const int64_t D = (int64_t)n * k;
  const int groups = (nsamples + SPW - 1) / SPW + 1;
  const int chunks = bn * CPR;
  const int64_t warps = (int64_t)gridDim.x * (blockDim.x / 32);
  for (int64_t w = (int64_t)blockIdx.x * (blockDim.x / 32) + (threadIdx.x >> 5); w < T * groups; w += warps) {
    const int64_t t = w / groups;
    const int u = (int)(w - t * groups);
    const bool last = u == groups - 1;
    const int n0 = u * SPW;
    const int ns = last ? 1 : min(SPW, nsamples - n0);
    const int r = (int)(t / kb), j = (int)(t - (int64_t)r * kb);
    float ah[SPW], al[SPW];
#pragma unroll
    for (int q = 0; q < SPW; ++q) ah[q] = al[q] = 0.f;
    float bh = 0.f, bl = 0.f;
    for (int c = lane; c < chunks; c += 32) {
      const int i = c / CPR, l = 4 * (c - i * CPR);
      const int64_t e = (int64_t)(r * bn + i) * k + (int64_t)j * BK + l;
      const uint2 wr = __ldg(reinterpret_cast<const uint2 *>(W + e));
      const float wv[4] = {__uint_as_float(wr.x << 16), __uint_as_float(wr.x & 0xffff0000u),
                           __uint_as_float(wr.y << 16), __uint_as_float(wr.y & 0xffff0000u)};
#pragma unroll
      for (int q = 0; q < SPW; ++q) {
        if (q < ns) {
          const float *src = last ? g : G + (int64_t)(n0 + q) * D;
          const float4 gv4 = __ldg(reinterpret_cast<const float4 *>(src + e));
          const float gv[4] = {gv4.x, gv4.y, gv4.z, gv4.w};
#pragma unroll
          for (int x = 0; x < 4; ++x) {
            const float p = __fmul_rn(wv[x], gv[x]);
            const float pe = __fmaf_rn(wv[x], gv[x], -p);  // w * g = p + pe exactly
            pair_add(ah[q], al[q], p);
            al[q] = __fadd_rn(al[q], pe);
          }
        }
      }
      if (last) {
#pragma unroll
        for (int x = 0; x < 4; ++x) pair_add(bh, bl, __fmul_rn(wv[x], wv[x]));  // a bf16 square is exact
      }
    }
#pragma unroll
    for (int q = 0; q < SPW; ++q) {
      if (q < ns) {
        warp_pair_sum(ah[q], al[q]);
        if (lane == 0) {
          if (last) gw[t] = make_float2(ah[q], al[q]);
          else s[(int64_t)(n0 + q) * T + t] = make_float2(ah[q], al[q]);
        }
      }
    }
    if (last) {
      warp_pair_sum(bh, bl);
      if (lane == 0) w2[t] = make_float2(bh, bl);
    }
  }
}

__device__ __forceinline__ int64_t prune_count_dev(int k, int steps, int64_t total) {
  const double alpha = (double)k / (double)steps;
  return (int64_t)floor(alpha * (double)total + 0.5);
}

__global__ void __launch_bounds__(ALLOC_THREADS)
order_kernel(const int32_t *__restrict__ rank, int64_t T, int32_t *__restrict__ order) {
  for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < T; t += (int64_t)gridDim.x * blockDim.x) {
    const int32_t rk = rank[t];
    if (rk >= 0 && rk < T) order[rk] = (int32_t)t;
  }
}

// Warp w handles step kk = 1 + w / (N + 1) and row u = w % (N + 1). The blocks newly pruned at
// step kk are those of rank [keep_kk, keep_{kk-1}): q[kk-1][u] = -sum s[u][t] over them (u < N);
// for u == N, lin[kk-1] = -sum gw[t] and sq[kk-1] = sum w2[t].
__global__ void __launch_bounds__(ALLOC_THREADS)
step_sums_kernel(const int32_t *__restrict__ order, const float2 *__restrict__ s, const float2 *__restrict__ gw,
                 const float2 *__restrict__ w2, int64_t T, int nsamples, int steps, double *__restrict__ q,
                 double *__restrict__ lin, double *__restrict__ sq) {
  const int lane = threadIdx.x & 31;
  const int64_t warps = (int64_t)gridDim.x * (blockDim.x / 32);
  for (int64_t w = (int64_t)blockIdx.x * (blockDim.x / 32) + (threadIdx.x >> 5);
       w < (int64_t)steps * (nsamples + 1); w += warps) {
    const int kk = 1 + (int)(w / (nsamples + 1));
    const int u = (int)(w - (int64_t)(kk - 1) * (nsamples + 1));
    const int64_t hi = T - prune_count_dev(kk - 1, steps, T), lo = T - prune_count_dev(kk, steps, T);
    float ah = 0.f, al = 0.f, ch = 0.f, cl = 0.f;
    for (int64_t rr = lo + lane; rr < hi; rr += 32) {
      const int32_t t = order[rr];
      const float2 v = u < nsamples ? s[(int64_t)u * T + t] : gw[t];
      pair_add2(ah, al, v.x, v.y);
      if (u == nsamples) {
        const float2 c = w2[t];
        pair_add2(ch, cl, c.x, c.y);
      }
    }
    warp_pair_sum(ah, al);
    if (u < nsamples) {
      if (lane == 0) q[(int64_t)(kk - 1) * nsamples + u] = -((double)ah + (double)al);
    } else {
      warp_pair_sum(ch, cl);
      if (lane == 0) {
        lin[kk - 1] = -((double)ah + (double)al);
        sq[kk - 1] = (double)ch + (double)cl;
      }
    }
  }
}

// CTA kk - 1 (one warp) computes step kk's increment of delta (see the file comment).
__global__ void __launch_bounds__(32)
increment_kernel(const double *__restrict__ q, const double *__restrict__ lin, const double *__restrict__ sq,
                 int nsamples, double kappa, double *__restrict__ inc) {
  const int kk = blockIdx.x + 1, lane = threadIdx.x;
  double qq = 0.0, pq = 0.0;
  for (int nn = lane; nn < nsamples; nn += 32) {
    double p = 0.0;
    for (int j = 0; j < kk - 1; ++j) p += q[(int64_t)j * nsamples + nn];
    const double qv = q[(int64_t)(kk - 1) * nsamples + nn];
    qq = fma(qv, qv, qq);
    pq = fma(p, qv, pq);
  }
  qq = warp_sum(qq);
  pq = warp_sum(pq);
  if (lane == 0) inc[kk - 1] = lin[kk - 1] + 0.5 * (kappa * sq[kk - 1] + qq / (double)nsamples) + pq / (double)nsamples;
}

__global__ void __launch_bounds__(32) prefix_kernel(const double *__restrict__ inc, int steps,
                                                    double *__restrict__ delta) {
  if (threadIdx.x != 0) return;
  double d = 0.0;
  delta[0] = 0.0;
  for (int kk = 1; kk <= steps; ++kk) {
    d += inc[kk - 1];
    delta[kk] = d;
  }
}

bool aligned_to(const void *p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }
bool side_ok(int v) { return v == 16 || v == 32 || v == 64; }
size_t round256(size_t v) { return (v + 255) / 256 * 256; }

struct AllocLayout {
  size_t g, scores, rank, order, s, gw, w2, q, lin, sq, inc, total;
};

AllocLayout alloc_layout(int nsamples, int n, int k, int bn, int bk, int steps) {
  const int64_t D = (int64_t)n * k, T = (int64_t)(n / bn) * (k / bk);
  AllocLayout L;
  size_t off = 0;
  L.g = off; off += round256(4 * (size_t)D);
  L.scores = off; off += round256(8 * (size_t)T);
  L.rank = off; off += round256(4 * (size_t)T);
  L.order = off; off += round256(4 * (size_t)T);
  L.s = off; off += round256(8 * (size_t)T * nsamples);  // float pairs
  L.gw = off; off += round256(8 * (size_t)T);
  L.w2 = off; off += round256(8 * (size_t)T);
  L.q = off; off += round256(8 * (size_t)steps * nsamples);
  L.lin = off; off += round256(8 * (size_t)steps);
  L.sq = off; off += round256(8 * (size_t)steps);
  L.inc = off; off += round256(8 * (size_t)steps);
  L.total = off;
  return L;
}

bool curve_args_ok(int nsamples, int n, int k, int bn, int bk) {
  return nsamples >= 1 && nsamples <= MAX_SAMPLES && n > 0 && k > 0 && n <= 65536 && k <= 65536 && side_ok(bn) &&
         side_ok(bk) && n % bn == 0 && k % bk == 0 && (int64_t)(n / bn) * (k / bk) <= MAX_ALLOC_BLOCKS;
}

}  // namespace
}  // namespace lpvit

using namespace lpvit;

extern "C" {

lpvit_status lpvit_mean_gradient(const float *G, int32_t nsamples, int64_t count, float *g, void *stream) {
  if (nsamples < 1 || nsamples > MAX_SAMPLES || count < 1 || !G || !g) return LPVIT_ERR_INVALID_ARG;
  if (!aligned_to(G, 4) || !aligned_to(g, 4)) return LPVIT_ERR_INVALID_ARG;
  const int64_t grid = (count + ALLOC_THREADS - 1) / ALLOC_THREADS;
  mean_grad_kernel<<<(int)(grid < 152 * 32 ? grid : 152 * 32), ALLOC_THREADS, 0, static_cast<cudaStream_t>(stream)>>>(
      G, nsamples, count, g);
  return cudaGetLastError() == cudaSuccess ? LPVIT_OK : LPVIT_ERR_CUDA;
}

size_t lpvit_delta_curve_workspace_bytes(int32_t nsamples, int32_t n, int32_t k, int32_t bn, int32_t bk,
                                         int32_t steps) {
  if (!curve_args_ok(nsamples, n, k, bn, bk) || steps < 1 || steps > MAX_STEPS) return 0;
  return alloc_layout(nsamples, n, k, bn, bk, steps).total;
}

lpvit_status lpvit_delta_curve(const void *W, const float *G, int32_t nsamples, int32_t n, int32_t k, int32_t bn,
                               int32_t bk, double kappa, int32_t steps, double *delta, void *workspace,
                               size_t ws_bytes, void *stream) {
  if (!side_ok(bn) || !side_ok(bk)) return LPVIT_ERR_UNSUPPORTED;
  if (n > 0 && k > 0 && n % bn == 0 && k % bk == 0 && (int64_t)(n / bn) * (k / bk) > MAX_ALLOC_BLOCKS)
    return LPVIT_ERR_UNSUPPORTED;
  if (!curve_args_ok(nsamples, n, k, bn, bk)) return LPVIT_ERR_INVALID_ARG;
  if (steps < 1 || steps > MAX_STEPS || !(kappa >= 0.0) || std::isinf(kappa)) return LPVIT_ERR_INVALID_ARG;
  if (!W || !G || !delta || !workspace) return LPVIT_ERR_INVALID_ARG;
  if (!aligned_to(W, 16) || !aligned_to(G, 16) || !aligned_to(delta, 8) || !aligned_to(workspace, 256))
    return LPVIT_ERR_INVALID_ARG;
  const AllocLayout L = alloc_layout(nsamples, n, k, bn, bk, steps);
  if (ws_bytes < L.total) return LPVIT_ERR_WORKSPACE;
  uint8_t *ws = static_cast<uint8_t *>(workspace);
  float *g = reinterpret_cast<float *>(ws + L.g);
  double *scores = reinterpret_cast<double *>(ws + L.scores);
  int32_t *rank = reinterpret_cast<int32_t *>(ws + L.rank);
  int32_t *order = reinterpret_cast<int32_t *>(ws + L.order);
  float2 *s = reinterpret_cast<float2 *>(ws + L.s);
  float2 *gw = reinterpret_cast<float2 *>(ws + L.gw);
  float2 *w2 = reinterpret_cast<float2 *>(ws + L.w2);
  double *inc = reinterpret_cast<double *>(ws + L.inc);
  double *q = reinterpret_cast<double *>(ws + L.q);
  double *lin = reinterpret_cast<double *>(ws + L.lin);
  double *sq = reinterpret_cast<double *>(ws + L.sq);
  const int64_t D = (int64_t)n * k, T = (int64_t)(n / bn) * (k / bk);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const uint16_t *Wh = static_cast<const uint16_t *>(W);
  int64_t grid = (D + ALLOC_THREADS - 1) / ALLOC_THREADS;
  mean_grad_kernel<<<(int)(grid < 152 * 32 ? grid : 152 * 32), ALLOC_THREADS, 0, st>>>(G, nsamples, D, g);
  if (cudaGetLastError() != cudaSuccess) return LPVIT_ERR_CUDA;
  if (launch_block_scores(Wh, g, n, k, bn, bk, scores, st) != cudaSuccess) return LPVIT_ERR_CUDA;
  if (launch_block_rank(scores, T, T, nullptr, rank, st) != cudaSuccess) return LPVIT_ERR_CUDA;
  grid = (T + ALLOC_THREADS - 1) / ALLOC_THREADS;
  order_kernel<<<(int)(grid < 152 * 8 ? grid : 152 * 8), ALLOC_THREADS, 0, st>>>(rank, T, order);
  if (cudaGetLastError() != cudaSuccess) return LPVIT_ERR_CUDA;
  const int64_t warps = T * ((nsamples + SPW - 1) / SPW + 1);
  grid = (warps + ALLOC_THREADS / 32 - 1) / (ALLOC_THREADS / 32);
  const int bgrid = (int)(grid < 152 * 64 ? grid : 152 * 64);
  switch (bk) {
    case 16: block_sums_kernel<16><<<bgrid, ALLOC_THREADS, 0, st>>>(Wh, G, g, nsamples, n, k, bn, s, gw, w2); break;
    case 32: block_sums_kernel<32><<<bgrid, ALLOC_THREADS, 0, st>>>(Wh, G, g, nsamples, n, k, bn, s, gw, w2); break;
    default: block_sums_kernel<64><<<bgrid, ALLOC_THREADS, 0, st>>>(Wh, G, g, nsamples, n, k, bn, s, gw, w2); break;
  }
  if (cudaGetLastError() != cudaSuccess) return LPVIT_ERR_CUDA;
  const int64_t swarps = (int64_t)steps * (nsamples + 1);
  grid = (swarps + ALLOC_THREADS / 32 - 1) / (ALLOC_THREADS / 32);
  step_sums_kernel<<<(int)(grid < 152 * 64 ? grid : 152 * 64), ALLOC_THREADS, 0, st>>>(order, s, gw, w2, T, nsamples,
                                                                                       steps, q, lin, sq);
  if (cudaGetLastError() != cudaSuccess) return LPVIT_ERR_CUDA;
  increment_kernel<<<steps, 32, 0, st>>>(q, lin, sq, nsamples, kappa, inc);
  if (cudaGetLastError() != cudaSuccess) return LPVIT_ERR_CUDA;
  prefix_kernel<<<1, 32, 0, st>>>(inc, steps, delta);
  return cudaGetLastError() == cudaSuccess ? LPVIT_OK : LPVIT_ERR_CUDA;
}

lpvit_status lpvit_lambda_search(int32_t layers, int32_t steps, const double *delta, const double *flops,
                                 const double *power_coef, double beta, double flops_ratio, int32_t *k_out,
                                 double *lambda_out, double *ratio_out) {
  if (layers < 1 || steps < 1 || steps > MAX_STEPS || !delta || !flops || !power_coef || !k_out)
    return LPVIT_ERR_INVALID_ARG;
  if (!std::isfinite(beta) || std::isnan(flops_ratio)) return LPVIT_ERR_INVALID_ARG;
  double ftot = 0.0;
  for (int i = 0; i < layers; ++i) {
    if (!(flops[i] > 0.0) || !std::isfinite(flops[i]) || !std::isfinite(power_coef[i])) return LPVIT_ERR_INVALID_ARG;
    ftot += flops[i];
  }
  // shifted slopes t[i][j] = (D_i[j+1] - D_i[j]) * steps - beta * c_i with D = delta^2 (Eq. obj_f)
  std::vector<double> t((size_t)layers * steps);
  for (int i = 0; i < layers; ++i)
    for (int j = 0; j < steps; ++j) {
      const double d1 = delta[(size_t)i * (steps + 1) + j + 1], d0 = delta[(size_t)i * (steps + 1) + j];
      const double v = (d1 * d1 - d0 * d0) * steps - beta * power_coef[i];
      if (std::isnan(v)) return LPVIT_ERR_INVALID_ARG;
      t[(size_t)i * steps + j] = v;
    }
  std::vector<double> cand(t);
  std::sort(cand.begin(), cand.end());
  cand.erase(std::unique(cand.begin(), cand.end()), cand.end());
  cand.insert(cand.begin(), -INFINITY);
  std::vector<int32_t> ks((size_t)layers);
  double lam = -INFINITY, ratio = 1.0;
  for (size_t c = 0; c < cand.size(); ++c) {
    lam = cand[c];
    double num = 0.0;
    for (int i = 0; i < layers; ++i) {
      int kk = 0;
      while (kk < steps && t[(size_t)i * steps + kk] <= lam) ++kk;
      ks[(size_t)i] = kk;
      num += (1.0 - (double)kk / (double)steps) * flops[i];
    }
    ratio = num / ftot;
    if (ratio <= flops_ratio) break;
  }
  for (int i = 0; i < layers; ++i) k_out[i] = ks[(size_t)i];
  if (lambda_out) *lambda_out = lam;
  if (ratio_out) *ratio_out = ratio;
  return LPVIT_OK;
}

}  // extern "C"
