// The non-linear parts of a pre-norm ViT (DeiT) encoder block around the block-sparse linears, so
// that a whole encoder forward runs in this library's kernels: residual add + LayerNorm, and
// multi-head softmax attention.
//
// add_layernorm_kernel (one warp per token row, 16-byte vectors): s = bf16(x + r) (x alone when r
//   is null), then y = (s - mean) / sqrt(var + eps) * gamma + beta over the row in float32 (biased
//   variance, two passes over the row held in registers), stored as bf16; s is stored too when r
//   is given (the new residual stream).
// attention_kernel (one CTA of ATT_WARPS = 7 warps per image and head; head_dim 64, at most 208
//   tokens): Q, K and V of the head are staged in shared memory by asynchronous 16-byte copies (rows
//   padded to 144 bytes: ldmatrix rows fall in distinct banks); each warp takes 16-query tiles in
//   turn (13 tiles for 197 tokens, two rounds). Per tile the keys stream in chunks of 64 with an
//   online softmax: S = Q K^T for the chunk with bf16 tensor-core MMAs (mma.sync m16n8k16, fp32
//   accumulation), scaled by 1/sqrt(64) (folded into base-2 exponentials), padded keys masked,
//   the running row max and sum updated over the four lanes sharing a row and the partial output
//   rescaled when the max grows; P = exp(S - max) rounded to bf16 is the A operand of O += P V (V
//   fragments by ldmatrix.trans); O / sum is stored as bf16. Attention is about 8% of the FLOPs of a
//   DeiT-B layer at 50% block density (30.5 GFLOP per layer at batch 256); these warp-level MMAs
//   are the legacy tensor path, kept because the kernel is latency-bound at 197 tokens per head.
#include <cmath>
#include <cstdint>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "lpvit.h"

namespace lpvit {

namespace {

constexpr int LN_THREADS = 256;
constexpr int LN_MAX_D = 1024;
constexpr int LN_VPL = LN_MAX_D / 8 / 32;  // 16-byte vectors per lane at most

constexpr int ATT_WARPS = 7;             // 13 query tiles of 16 in two rounds
constexpr int KCHUNK = 8;                // key tiles of 8 per online-softmax chunk (64 keys)
constexpr int HD = 64;                   // head dimension
constexpr int MAX_TOKENS = 208;          // 13 tiles of 16
constexpr int ROW = HD + 8;              // shared-memory row in bf16 (144 bytes)
constexpr int ATT_SMEM = 3 * MAX_TOKENS * ROW * 2;

__device__ __forceinline__ float warp_sum_f(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// A warp per row; the kernel is latency-bound (one 1.5 KB row per warp for D = 768), so its
// registers are held to 64 for four CTAs (32 warps) per SM.
__global__ void __launch_bounds__(LN_THREADS, 4)
add_layernorm_kernel(const __nv_bfloat16 *__restrict__ x, const __nv_bfloat16 *__restrict__ r,
                     const float *__restrict__ gamma, const float *__restrict__ beta, int64_t rows, int D, float eps,
                     __nv_bfloat16 *__restrict__ sum_out, __nv_bfloat16 *__restrict__ norm_out) {
  const int lane = threadIdx.x & 31;
  const int nv = D / 8;
  const int64_t warps = (int64_t)gridDim.x * (blockDim.x / 32);
  for (int64_t row = (int64_t)blockIdx.x * (blockDim.x / 32) + (threadIdx.x >> 5); row < rows; row += warps) {
    const int64_t base = row * D;
    float v[LN_VPL][8];
    float s1 = 0.f;
#pragma unroll
    for (int i = 0; i < LN_VPL; ++i) {
      const int c = lane + 32 * i;
      if (c < nv) {
        const uint4 xv = __ldg(reinterpret_cast<const uint4 *>(x + base) + c);
        const __nv_bfloat16 *xb = reinterpret_cast<const __nv_bfloat16 *>(&xv);
        uint4 sv = xv;
        if (r) {
          const uint4 rv = __ldg(reinterpret_cast<const uint4 *>(r + base) + c);
          const __nv_bfloat16 *rb = reinterpret_cast<const __nv_bfloat16 *>(&rv);
          __nv_bfloat16 *sb = reinterpret_cast<__nv_bfloat16 *>(&sv);
#pragma unroll
          for (int e = 0; e < 8; ++e) sb[e] = __float2bfloat16_rn(__bfloat162float(xb[e]) + __bfloat162float(rb[e]));
          reinterpret_cast<uint4 *>(sum_out + base)[c] = sv;
        }
        const __nv_bfloat16 *sb = reinterpret_cast<const __nv_bfloat16 *>(&sv);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          v[i][e] = __bfloat162float(sb[e]);
          s1 += v[i][e];
        }
      }
    }
    const float mean = warp_sum_f(s1) / (float)D;
    float s2 = 0.f;
#pragma unroll
    for (int i = 0; i < LN_VPL; ++i)
      if (lane + 32 * i < nv) {
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const float d = v[i][e] - mean;
          s2 += d * d;
        }
      }
    const float rstd = rsqrtf(warp_sum_f(s2) / (float)D + eps);
#pragma unroll
    for (int i = 0; i < LN_VPL; ++i) {
      const int c = lane + 32 * i;
      if (c < nv) {
        uint4 ov;
        __nv_bfloat16 *ob = reinterpret_cast<__nv_bfloat16 *>(&ov);
        const float4 g0 = __ldg(reinterpret_cast<const float4 *>(gamma) + 2 * c);
        const float4 g1 = __ldg(reinterpret_cast<const float4 *>(gamma) + 2 * c + 1);
        const float4 b0 = __ldg(reinterpret_cast<const float4 *>(beta) + 2 * c);
        const float4 b1 = __ldg(reinterpret_cast<const float4 *>(beta) + 2 * c + 1);
        const float gg[8] = {g0.x, g0.y, g0.z, g0.w, g1.x, g1.y, g1.z, g1.w};
        const float bb[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
        for (int e = 0; e < 8; ++e) ob[e] = __float2bfloat16_rn((v[i][e] - mean) * rstd * gg[e] + bb[e]);
        reinterpret_cast<uint4 *>(norm_out + base)[c] = ov;
      }
    }
  }
}

__device__ __forceinline__ uint32_t smem_addr(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t &a0, uint32_t &a1, uint32_t &a2, uint32_t &a3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(a0), "=r"(a1), "=r"(a2), "=r"(a3) : "r"(addr));
}
__device__ __forceinline__ void ldsm_x2(uint32_t addr, uint32_t &b0, uint32_t &b1) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.shared.b16 {%0,%1}, [%2];" : "=r"(b0), "=r"(b1) : "r"(addr));
}
__device__ __forceinline__ void ldsm_x2_trans(uint32_t addr, uint32_t &b0, uint32_t &b1) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.trans.shared.b16 {%0,%1}, [%2];" : "=r"(b0), "=r"(b1) : "r"(addr));
}
// D (16x8 fp32) += A (16x16 bf16, row) * B (16x8 bf16, col)
__device__ __forceinline__ void mma_bf16(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
  asm volatile("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
               "{%0,%1,%2,%3};"
               : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
               : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 p = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t *>(&p);
}

// One CTA per (image, head): Q, K, V of the head staged in shared memory by asynchronous copies;
// each warp takes 16-query tiles and streams the keys in chunks of 64 with an online softmax
// (running row max and sum, rescaling the partial output when the max grows), so a chunk's scores
// stay in 32 registers per thread. Scores and exponentials in float32 (base 2, the 1/sqrt(64) scale
// folded into log2 e), P rounded to bf16 for the P V products, fp32 accumulation.
__global__ void __launch_bounds__(32 * ATT_WARPS, 2)
attention_kernel(const __nv_bfloat16 *__restrict__ qkv, int tokens, int heads, __nv_bfloat16 *__restrict__ out) {
  extern __shared__ __align__(16) __nv_bfloat16 att_smem[];
  __nv_bfloat16 *Qs = att_smem, *Ks = Qs + MAX_TOKENS * ROW, *Vs = Ks + MAX_TOKENS * ROW;
  const int img = blockIdx.x / heads, h = blockIdx.x - img * heads;
  const int D = heads * HD;
  const int tp = (tokens + 15) / 16 * 16;  // padded token count
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // stage Q, K, V of this head (8 vectors of 16 bytes per row each) with asynchronous copies, all
  // in flight together; padded rows are zero
  for (int idx = threadIdx.x; idx < tp * 8 * 3; idx += blockDim.x) {
    const int m = idx / (tp * 8), rem = idx - m * tp * 8, row = rem >> 3, c = rem & 7;
    uint4 *dst = reinterpret_cast<uint4 *>(att_smem + (m * MAX_TOKENS + row) * ROW) + c;
    if (row < tokens) {
      const uint4 *src =
          reinterpret_cast<const uint4 *>(qkv + ((int64_t)img * tokens + row) * 3 * D + m * D + h * HD) + c;
      asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" :: "r"(smem_addr(dst)), "l"(src) : "memory");
    } else {
      *dst = make_uint4(0, 0, 0, 0);
    }
  }
  asm volatile("cp.async.wait_all;" ::: "memory");
  __syncthreads();
  constexpr float kScaleLog2 = 0.125f * 1.4426950408889634f;  // 1/sqrt(64) * log2(e)
  const int ntiles = tp / 8, kq = lane & 3, rq = lane >> 2;
  for (int mt = warp; mt < tp / 16; mt += ATT_WARPS) {
    uint32_t qa[HD / 16][4];
#pragma unroll
    for (int ks = 0; ks < HD / 16; ++ks)
      ldsm_x4(smem_addr(Qs + (16 * mt + (lane & 15)) * ROW + 16 * ks + (lane >> 4) * 8), qa[ks][0], qa[ks][1],
              qa[ks][2], qa[ks][3]);
    float o[HD / 8][4];
#pragma unroll
    for (int nd = 0; nd < HD / 8; ++nd) o[nd][0] = o[nd][1] = o[nd][2] = o[nd][3] = 0.f;
    float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;  // rows rq and rq + 8 of the tile
    for (int kc = 0; kc < ntiles; kc += KCHUNK) {
      // S = Q K^T for keys 8 kc .. 8 (kc + KCHUNK)
      float s[KCHUNK][4];
#pragma unroll
      for (int nt = 0; nt < KCHUNK; ++nt) {
        s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
        if (kc + nt < ntiles) {
#pragma unroll
          for (int ks = 0; ks < HD / 16; ++ks) {
            uint32_t b0, b1;
            ldsm_x2(smem_addr(Ks + (8 * (kc + nt) + (lane & 7)) * ROW + 16 * ks + ((lane >> 3) & 1) * 8), b0, b1);
            mma_bf16(s[nt], qa[ks][0], qa[ks][1], qa[ks][2], qa[ks][3], b0, b1);
          }
        }
      }
      float cm0 = -INFINITY, cm1 = -INFINITY;
#pragma unroll
      for (int nt = 0; nt < KCHUNK; ++nt) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int col = 8 * (kc + nt) + 2 * kq + (e & 1);
          s[nt][e] = col < tokens ? s[nt][e] * kScaleLog2 : -INFINITY;
        }
        cm0 = fmaxf(cm0, fmaxf(s[nt][0], s[nt][1]));
        cm1 = fmaxf(cm1, fmaxf(s[nt][2], s[nt][3]));
      }
      cm0 = fmaxf(cm0, __shfl_xor_sync(0xffffffffu, cm0, 1));
      cm0 = fmaxf(cm0, __shfl_xor_sync(0xffffffffu, cm0, 2));
      cm1 = fmaxf(cm1, __shfl_xor_sync(0xffffffffu, cm1, 1));
      cm1 = fmaxf(cm1, __shfl_xor_sync(0xffffffffu, cm1, 2));
      // the first chunk always holds key 0, so the running max is finite from here on
      const float n0 = fmaxf(m0, cm0), n1 = fmaxf(m1, cm1);
      const float a0 = exp2f(m0 - n0), a1 = exp2f(m1 - n1);  // 0 on the first chunk
      m0 = n0;
      m1 = n1;
      l0 *= a0;
      l1 *= a1;
#pragma unroll
      for (int nd = 0; nd < HD / 8; ++nd) {
        o[nd][0] *= a0;
        o[nd][1] *= a0;
        o[nd][2] *= a1;
        o[nd][3] *= a1;
      }
#pragma unroll
      for (int nt = 0; nt < KCHUNK; ++nt) {
        s[nt][0] = exp2f(s[nt][0] - n0);
        s[nt][1] = exp2f(s[nt][1] - n0);
        s[nt][2] = exp2f(s[nt][2] - n1);
        s[nt][3] = exp2f(s[nt][3] - n1);
        l0 += s[nt][0] + s[nt][1];
        l1 += s[nt][2] + s[nt][3];
      }
      // O += P V over the chunk's keys, 16 at a time (ntiles is even)
#pragma unroll
      for (int kt = 0; kt < KCHUNK / 2; ++kt) {
        if (kc + 2 * kt < ntiles) {
          const uint32_t p0 = pack_bf16(s[2 * kt][0], s[2 * kt][1]), p1 = pack_bf16(s[2 * kt][2], s[2 * kt][3]);
          const uint32_t p2 = pack_bf16(s[2 * kt + 1][0], s[2 * kt + 1][1]);
          const uint32_t p3 = pack_bf16(s[2 * kt + 1][2], s[2 * kt + 1][3]);
#pragma unroll
          for (int nd = 0; nd < HD / 8; ++nd) {
            uint32_t b0, b1;
            ldsm_x2_trans(smem_addr(Vs + (8 * kc + 16 * kt + (lane & 15)) * ROW + 8 * nd), b0, b1);
            mma_bf16(o[nd], p0, p1, p2, p3, b0, b1);
          }
        }
      }
    }
    l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
    l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
    const float inv0 = 1.f / l0, inv1 = 1.f / l1;
    const int r0 = 16 * mt + rq, r1 = r0 + 8;
#pragma unroll
    for (int nd = 0; nd < HD / 8; ++nd) {
      const int col = h * HD + 8 * nd + 2 * kq;
      if (r0 < tokens)
        *reinterpret_cast<uint32_t *>(out + ((int64_t)img * tokens + r0) * D + col) =
            pack_bf16(o[nd][0] * inv0, o[nd][1] * inv0);
      if (r1 < tokens)
        *reinterpret_cast<uint32_t *>(out + ((int64_t)img * tokens + r1) * D + col) =
            pack_bf16(o[nd][2] * inv1, o[nd][3] * inv1);
    }
  }
}

bool aligned_to(const void *p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

}  // namespace
}  // namespace lpvit

using namespace lpvit;

extern "C" {

lpvit_status lpvit_add_layernorm(const void *x, const void *r, const float *gamma, const float *beta, int64_t rows,
                                 int32_t D, double eps, void *sum_out, void *norm_out, void *stream) {
  if (rows < 0 || D < 8 || D > LN_MAX_D || D % 8 || !(eps > 0.0) || !std::isfinite(eps)) return LPVIT_ERR_INVALID_ARG;
  if (rows == 0) return LPVIT_OK;
  if (!x || !gamma || !beta || !norm_out || (r && !sum_out)) return LPVIT_ERR_INVALID_ARG;
  if (!aligned_to(x, 16) || !aligned_to(gamma, 16) || !aligned_to(beta, 16) || !aligned_to(norm_out, 16) ||
      (r && (!aligned_to(r, 16) || !aligned_to(sum_out, 16))))
    return LPVIT_ERR_INVALID_ARG;
  const int64_t want = (rows + LN_THREADS / 32 - 1) / (LN_THREADS / 32);
  const int grid = (int)(want < 152 * 32 ? want : 152 * 32);
  add_layernorm_kernel<<<grid, LN_THREADS, 0, static_cast<cudaStream_t>(stream)>>>(
      static_cast<const __nv_bfloat16 *>(x), static_cast<const __nv_bfloat16 *>(r), gamma, beta, rows, D, (float)eps,
      static_cast<__nv_bfloat16 *>(sum_out), static_cast<__nv_bfloat16 *>(norm_out));
  return cudaGetLastError() == cudaSuccess ? LPVIT_OK : LPVIT_ERR_CUDA;
}

lpvit_status lpvit_attention(const void *qkv, int64_t images, int32_t tokens, int32_t heads, int32_t head_dim,
                             void *out, void *stream) {
  if (head_dim != HD || tokens < 1 || tokens > MAX_TOKENS) return LPVIT_ERR_UNSUPPORTED;
  if (images < 0 || heads < 1 || heads > 64) return LPVIT_ERR_INVALID_ARG;
  if (images == 0) return LPVIT_OK;
  if (images * heads > 0x7fffffffLL) return LPVIT_ERR_INVALID_ARG;
  if (!qkv || !out || !aligned_to(qkv, 16) || !aligned_to(out, 16)) return LPVIT_ERR_INVALID_ARG;
  static bool attr_done[64] = {false};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64 && !attr_done[dev]) {
    if (cudaFuncSetAttribute(attention_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, ATT_SMEM) != cudaSuccess)
      return LPVIT_ERR_CUDA;
    attr_done[dev] = true;
  }
  attention_kernel<<<(int)(images * heads), 32 * ATT_WARPS, ATT_SMEM, static_cast<cudaStream_t>(stream)>>>(
      static_cast<const __nv_bfloat16 *>(qkv), tokens, heads, static_cast<__nv_bfloat16 *>(out));
  return cudaGetLastError() == cudaSuccess ? LPVIT_OK : LPVIT_ERR_CUDA;
}

}  // extern "C"
