// The non-linear parts of a pre-norm ViT (DeiT) encoder block around the block-sparse linears, so
// that a whole encoder forward runs in this library's kernels: residual add + LayerNorm, and
// multi-head softmax attention.
//
// add_layernorm_kernel (one warp per token row, 16-byte vectors): s = bf16(x + r) (x alone when r
//   is null), then y = (s - mean) / sqrt(var + eps) * gamma + beta over the row in float32 (biased
//   variance, two passes over the row held in registers), stored as bf16; s is stored too when r
//   is given (the new residual stream).
// attention_kernel (tcgen05; one CTA of four warps per image, head and 128-query tile; head_dim 64,
//   at most 208 tokens): the tile's Q rows and the head's K rows are copied by 16-byte cp.async into
//   K-major tiles of 128-byte rows in the 128-byte swizzle, V's rows as they are; while the first
//   MMAs run, the threads transpose V in shared memory into K-major tiles (the 64 dims as rows, keys
//   along K, two keys per 32-bit store). S = Q K^T is four tcgen05 MMAs (M = 128
//   queries, N = the keys rounded up to 16, K = 16) into TMEM; each thread then takes one query row
//   of S from TMEM: the row max over the valid keys, p = 2^((s - max) log2(e) / sqrt(64)) for them
//   (ex2.approx.ftz; 0 for padding keys), their float32 sum, and p rounded to bf16 into the K-major P tiles (written
//   over Q, K and V's rows, no longer read). O = P V is one MMA per 16 keys (N = 64)
//   into the first TMEM columns, where S was; O / sum is rounded to bf16 and stored. Attention is
//   about 8% of the FLOPs of a DeiT-B layer at 50% block density (30.5 GFLOP per layer at batch 256).
#include <cmath>
#include <cstdint>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "lpvit.h"
#include "lpvit_device.cuh"

namespace lpvit {

namespace {

constexpr int LN_THREADS = 256;
constexpr int LN_MAX_D = 1024;
constexpr int LN_VPL = LN_MAX_D / 8 / 32;  // 16-byte vectors per lane at most

constexpr int HD = 64;                      // head dimension
constexpr int MAX_TOKENS = 208;             // 13 key tiles of 16
constexpr int AT_Q = 128;                   // queries per CTA: the MMA's M, one TMEM lane each
constexpr int AT_THREADS = 128;
constexpr int AT_K_OFF = AT_Q * 128;        // K's rows after the 128 Q rows
constexpr int AT_V_OFF = AT_K_OFF + MAX_TOKENS * 128;  // V's rows as they are (128-byte rows)
constexpr int AT_P_CHUNK = AT_Q * 128;      // P: four 64-key chunks of [128 rows x 128 bytes], from 0
constexpr int AT_VT_OFF = 68 * 1024;        // V^T: four 64-key chunks of [64 dims x 128 bytes]
constexpr int AT_VT_CHUNK = HD * 128;
constexpr int AT_TMEM_COLS = 256;           // S (up to 208 columns); O reuses the first 64
constexpr int AT_SMEM = AT_VT_OFF + 4 * AT_VT_CHUNK + 1024;  // + alignment slack (101 KB: two CTAs per SM)
constexpr float AT_SCALE_LOG2 = 0.125f * 1.4426950408889634f;  // 1/sqrt(64) * log2(e)
constexpr uint64_t AT_WAIT_NS = 2000000000ull;
static_assert(AT_V_OFF + MAX_TOKENS * 128 <= AT_VT_OFF && 4 * AT_P_CHUNK <= AT_VT_OFF, "Q, K, V and P before V^T");

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

// V's staged rows: piece j of key row r at j ^ ((r / 2) mod 8), so that the transpose's reads of one
// piece of 32 consecutive even (or odd) keys fall in distinct bank groups.
__device__ __forceinline__ uint32_t v_off(int r, int j) { return (uint32_t)(r * 128 + ((j ^ ((r >> 1) & 7)) << 4)); }
__device__ __forceinline__ float ex2_ftz(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Grid: images x heads x ceil(tokens / 128) CTAs; qkv [images * tokens][3 D] (q | k | v, head h at
// columns h * 64 of each), out [images * tokens][D], D = heads * 64.
__global__ void __launch_bounds__(AT_THREADS)
attention_kernel(const __nv_bfloat16 *__restrict__ qkv, int tokens, int heads, __nv_bfloat16 *__restrict__ out) {
  extern __shared__ uint8_t at_raw[];
  uint8_t *sm = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(at_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t bars[2];
  __shared__ uint32_t tmem_slot;
  __shared__ int abort_flag;  // stays 0: the waits end by completion or their time limit
  const uint32_t base = smem_u32(sm);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nqt = (tokens + AT_Q - 1) / AT_Q;
  const int qt = (int)(blockIdx.x % (unsigned)nqt);
  const int bh = (int)(blockIdx.x / (unsigned)nqt);
  const int img = bh / heads, h = bh - img * heads;
  const int D = heads * HD;
  const int64_t row0 = (int64_t)img * tokens;  // the image's first token row
  const int64_t ld = 3 * (int64_t)D;           // elements per qkv row
  const int nkeys = (tokens + 15) & ~15;       // S's N
  const uint32_t bar_s = smem_u32(&bars[0]), bar_o = smem_u32(&bars[1]);

  if (warp == 0) {
    tmem_alloc(smem_u32(&tmem_slot), AT_TMEM_COLS);
    tmem_relinquish();
  }
  if (tid == 0) {
    mbar_init(bar_s, 1);
    mbar_init(bar_o, 1);
    abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  // the tile's Q rows and the head's K rows (zero past the tokens)
  for (int pc = tid; pc < AT_Q * 8; pc += AT_THREADS) {
    const int r = pc >> 3, j = pc & 7, t = qt * AT_Q + r;
    const bool in = t < tokens;
    cp_async16(base + sw_off(r, j), qkv + (in ? (row0 + t) * ld + h * HD + j * 8 : 0), in ? 16u : 0u);
  }
  for (int pc = tid; pc < nkeys * 8; pc += AT_THREADS) {
    const int r = pc >> 3, j = pc & 7;
    const bool in = r < tokens;
    cp_async16(base + AT_K_OFF + sw_off(r, j), qkv + (in ? (row0 + r) * ld + D + h * HD + j * 8 : 0), in ? 16u : 0u);
  }
  for (int pc = tid; pc < nkeys * 8; pc += AT_THREADS) {
    const int r = pc >> 3, j = pc & 7;
    const bool in = r < tokens;
    cp_async16(base + AT_V_OFF + v_off(r, j), qkv + (in ? (row0 + r) * ld + 2 * D + h * HD + j * 8 : 0),
               in ? 16u : 0u);
  }
  cp_async_commit();
  cp_async_wait<0>();
  fence_proxy_async_smem();  // this thread's copies, visible to the tensor core
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_slot;
  if (tid == 0) {
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk)
      umma_f16(tmem, smem_desc<128>(base + kk * 32), smem_desc<128>(base + AT_K_OFF + kk * 32),
               idesc_bf16(AT_Q, nkeys), kk > 0 ? 1u : 0u);
    tc_commit(bar_s);
  }
  // V^T while S is computed: dims 8 dp .. 8 dp + 7 of keys r, r + 1 become columns r, r + 1 of rows
  // 8 dp .. 8 dp + 7 of key chunk r / 64 (consecutive threads take consecutive key pairs)
  for (int it = tid; it < 4 * nkeys; it += AT_THREADS) {
    const int dp = it / (nkeys / 2), r = 2 * (it - dp * (nkeys / 2));
    uint4 a, b;
    asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];" : "=r"(a.x), "=r"(a.y), "=r"(a.z), "=r"(a.w)
                 : "r"(base + AT_V_OFF + v_off(r, dp)));
    asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];" : "=r"(b.x), "=r"(b.y), "=r"(b.z), "=r"(b.w)
                 : "r"(base + AT_V_OFF + v_off(r + 1, dp)));
    const uint32_t wa[4] = {a.x, a.y, a.z, a.w}, wb[4] = {b.x, b.y, b.z, b.w};
    const uint32_t col = base + AT_VT_OFF + (r >> 6) * AT_VT_CHUNK + 2 * (r & 7);
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const uint32_t lo = (e & 1) ? (wa[e >> 1] >> 16) : (wa[e >> 1] & 0xffffu);
      const uint32_t hi = (e & 1) ? (wb[e >> 1] >> 16) : (wb[e >> 1] & 0xffffu);
      asm volatile("st.shared.b32 [%0], %1;" :: "r"(col + sw_off(dp * 8 + e, (r & 63) >> 3)), "r"(lo | (hi << 16))
                   : "memory");
    }
  }
  __syncthreads();  // V's rows are read: P may be written over them
  bool ok = mbar_wait(bar_s, 0, &abort_flag, AT_WAIT_NS);
  tc_fence_after();

  // softmax of this thread's query row (TMEM lane r), in chunks of 32 keys
  const int r = 32 * warp + lane;
  const uint32_t trow = tmem + ((uint32_t)(32 * warp) << 16);
  const int nch = (nkeys + 31) / 32;
  float m = -INFINITY;
  for (int c = 0; c < nch; ++c) {
    float v[32];
    tmem_ld32(trow + 32 * c, v);
#pragma unroll
    for (int i = 0; i < 32; ++i)
      m = 32 * c + i < tokens ? fmaxf(m, v[i]) : m;
  }
  const float mb = m * AT_SCALE_LOG2;
  float sum = 0.f;
  for (int c = 0; c < nch; ++c) {
    float v[32];
    tmem_ld32(trow + 32 * c, v);
    uint32_t pk[16];
    const bool full = 32 * c + 32 <= tokens;  // warp-uniform: only the last chunk holds padding keys
#pragma unroll
    for (int i = 0; i < 32; i += 2) {
      float p0 = ex2_ftz(fmaf(v[i], AT_SCALE_LOG2, -mb)), p1 = ex2_ftz(fmaf(v[i + 1], AT_SCALE_LOG2, -mb));
      if (!full) {
        p0 = 32 * c + i < tokens ? p0 : 0.f;
        p1 = 32 * c + i + 1 < tokens ? p1 : 0.f;
      }
      sum += p0 + p1;
      asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(pk[i / 2]) : "f"(p1), "f"(p0));
    }
    // keys 32 c .. 32 c + 31: chunk c / 2, 16-byte pieces 4 (c % 2) .. 4 (c % 2) + 3 of row r
    const uint32_t prow = base + (c >> 1) * AT_P_CHUNK;
#pragma unroll
    for (int q = 0; q < 4; ++q)
      asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(prow + sw_off(r, (c & 1) * 4 + q)),
                   "r"(pk[4 * q]), "r"(pk[4 * q + 1]), "r"(pk[4 * q + 2]), "r"(pk[4 * q + 3]) : "memory");
  }
  fence_proxy_async_smem();
  tc_fence_before();  // every thread's S loads are complete: O may overwrite those columns
  __syncthreads();
  tc_fence_after();
  if (tid == 0) {
    for (int st = 0; st < nkeys / 16; ++st) {
      const int c = st >> 2, kk = st & 3;
      umma_f16(tmem, smem_desc<128>(base + c * AT_P_CHUNK + kk * 32),
               smem_desc<128>(base + AT_VT_OFF + c * AT_VT_CHUNK + kk * 32), idesc_bf16(AT_Q, HD),
               st > 0 ? 1u : 0u);
    }
    tc_commit(bar_o);
  }
  ok = mbar_wait(bar_o, 0, &abort_flag, AT_WAIT_NS) && ok;
  tc_fence_after();

  const int t = qt * AT_Q + r;
  const float inv = 1.f / sum;
#pragma unroll
  for (int half = 0; half < 2; ++half) {
    float o[32];
    tmem_ld32(trow + 32 * half, o);
    if (ok && t < tokens) {
      uint32_t w[16];
#pragma unroll
      for (int i = 0; i < 16; ++i)
        asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(w[i]) : "f"(o[2 * i + 1] * inv), "f"(o[2 * i] * inv));
      uint4 *dst = reinterpret_cast<uint4 *>(out + (row0 + t) * D + h * HD + half * 32);
#pragma unroll
      for (int q = 0; q < 4; ++q) dst[q] = make_uint4(w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, AT_TMEM_COLS);
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
  const int64_t ctas = images * heads * ((tokens + AT_Q - 1) / AT_Q);
  if (ctas > 0x7fffffffLL) return LPVIT_ERR_INVALID_ARG;
  if (!qkv || !out || !aligned_to(qkv, 16) || !aligned_to(out, 16)) return LPVIT_ERR_INVALID_ARG;
  static bool attr_done[64] = {false};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64 && !attr_done[dev]) {
    if (cudaFuncSetAttribute(attention_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, AT_SMEM) != cudaSuccess)
      return LPVIT_ERR_CUDA;
    attr_done[dev] = true;
  }
  attention_kernel<<<(int)ctas, AT_THREADS, AT_SMEM, static_cast<cudaStream_t>(stream)>>>(
      static_cast<const __nv_bfloat16 *>(qkv), tokens, heads, static_cast<__nv_bfloat16 *>(out));
  return cudaGetLastError() == cudaSuccess ? LPVIT_OK : LPVIT_ERR_CUDA;
}

}  // extern "C"
