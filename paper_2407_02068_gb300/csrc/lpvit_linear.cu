// Block-sparse linear Y = act(X W~^T + bias) on sm_103a (Sec. 3.1 block mask, Sec. 3.3
// block-sparse matmul: work for the kept blocks; tiles whose blocks are all removed are skipped).
//
// Work unit = 256 tokens x one group of 256 output features (x one slice of the group's entries
// when the problem is too small to fill the GPU). A unit runs on a CTA pair (cluster of two CTAs on
// two SMs) with tcgen05 MMAs of cta_group::2: M = 256 tokens (128 per CTA, the A operand), N = 256
// features (128 weight rows staged per CTA, the B operand), K = 16, fp32 accumulators in TMEM
// (each CTA holds its 128 tokens x 256 features). Per work-list entry, one chunk of 64 input
// columns: a stage of two tensor copies per CTA (its 128 x 64 X tile and its 128 x 64 half of the
// entry's weight-stream tile, 128-byte swizzle), four MMAs.
// Per CTA (one per SM, persistent):
//   warp 0      X producer: walks each unit's entries and loads its X tiles, two stages per batch,
//               every copy completing on the leader's full barrier.
//   warp 18     weight producer: the same walk, loading the weight tiles (a second issuing warp:
//               a tensor copy keeps its issuing thread for a few hundred cycles).
//   warp 19     scheduler (leader only): takes units (pair p's first unit is unit p, the rest come
//               from a global atomic queue) and publishes each,
//               with the chunk indices of its first 32 entries, to both CTAs' unit rings, up to
//               UR units ahead of the producers.
//   warp 1      MMA issuer (leader only): per stage four MMAs, the commit multicast to both CTAs'
//               empty barriers; per unit the commit to both CTAs' accumulator-full barriers.
//   warps 2..17 epilogue: TMEM -> registers (a lane per token, consecutive features along the
//               registers), + bias, optional exact GELU, rounding, optional bf16 residual, stores
//               of whole 16-byte pieces of output rows; split units write fp32 partial sums that
//               the reduction kernel adds in slice order (deterministic).
// Accumulators are double-buffered in TMEM (2 x 256 columns), so one unit's epilogue overlaps the
// next unit's MMAs. Every wait is bounded: on timeout the CTA records an error bit, drains its own
// copies and MMAs, frees TMEM and returns.
// A chain launch runs several linears over the same tokens in one launch (units of linear j after
// those of linear j - 1): each CTA counts a unit's stores on a per-(linear, token tile) counter with
// a gpu-scope release, and the X producer of a unit of linear j waits (acquire, then a proxy fence)
// for linear j - 1's count on its token tile before its tensor copies. No launch boundary separates
// the linears: one linear's last units overlap the next one's first.
#include <cstddef>
#include <cstdint>
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "lpvit_device.cuh"

namespace lpvit {

namespace {

// Stages of the copy pipeline: six when the epilogue stages its bias in shared memory, seven when it
// reads the bias from the L1-cached global copy instead (the fourth kilobyte of that staging is what
// a seventh stage needs). Long-K launches (many entries per unit) are bound by the copy feed and take
// the deeper ring; short-K launches are bound by their epilogue and keep the staged bias.
template <bool DEEP> struct Depth { static constexpr int NSTAGES = DEEP ? 7 : 6; };
constexpr int X_BYTES = CTA_TOKENS * CHUNK_COLS * 2;      // 16 KB: this CTA's tokens x 64 columns
constexpr int W_BYTES = HALF_FEATURES * CHUNK_COLS * 2;   // 16 KB: this CTA's weight rows x 64 columns
constexpr int STAGE_BYTES = X_BYTES + W_BYTES;
constexpr int KSTEPS = CHUNK_COLS / 16;
constexpr int BUF_COLS = GROUP_FEATURES;                  // TMEM columns of one accumulator
constexpr int DEEP_MIN_CHUNKS = 24;                       // units of >= 24 entries take seven stages
constexpr int UR = 3;                                     // unit ring depth: units are handed out at most
                                                          // three ahead, so the queue's last units stay balanced
constexpr int BATCH = 2;                                  // stages per producer batch
static_assert(32 % BATCH == 0, "producer batches tile the 32-entry windows");
constexpr int FIRST_EPI = 2;
constexpr int EPI_WARPS = 16;                             // four per TMEM lane quarter
constexpr int W_WARP = FIRST_EPI + EPI_WARPS;             // the weight-copy producer
constexpr int SCHED_WARP = W_WARP + 1;                    // the pair's unit scheduler (leader)
constexpr int NUM_THREADS = 32 * (SCHED_WARP + 1);        // 640
constexpr int MAX_GROUPS = 256;                           // n <= 65536
constexpr uint32_t IDESC = idesc_bf16(2 * CTA_TOKENS, GROUP_FEATURES);
// arrivals that free a unit-ring slot: the leader's MMA warp, both CTAs' epilogue warps and both
// CTAs' two producers
constexpr int UNIT_CONSUMERS = 1 + 2 * EPI_WARPS + 4;
static_assert(2 * BUF_COLS == 512, "two accumulator buffers fill the 512 TMEM columns");
static_assert(CHUNK_COLS * 2 == 128, "stage rows are 128 bytes (the 128-byte swizzle)");
static_assert(EPI_WARPS == 16 && GROUP_FEATURES == 4 * 64, "each epilogue warp takes 64 feature columns");

struct UnitInfo {
  int tt, g, s, nsl, e0, e1;
  int ptile;  // split units: the partial tile (token tile, group slice) the slice writes
  int pad;
};
static_assert(sizeof(UnitInfo) == 32, "unit record is two 16-byte vectors");
// A unit-ring slot: the unit and the chunk indices of its first 32 entries (0 past its end).
struct UnitSlot {
  UnitInfo inf;
  int win[32];
};

template <bool DEEP>
struct Smem {
  static constexpr int NSTAGES = Depth<DEEP>::NSTAGES;
  static constexpr int BAR_OFF = NSTAGES * STAGE_BYTES;
  // barriers: full[NS], empty[NS], accf[2], acce[2], unitf[UR], unite[UR], drain, stored[2] (chain)
  static constexpr int NBARS = 2 * NSTAGES + 4 + 2 * UR + 3;
  static constexpr int RING_OFF = (BAR_OFF + 8 * NBARS + 31) / 32 * 32;
  static constexpr int MISC_OFF = RING_OFF + (int)sizeof(UnitSlot) * UR;
  static constexpr int BIAS_OFF = MISC_OFF + 64;  // per epilogue warp: its 64 features' bias
  static constexpr int END = BIAS_OFF + (DEEP ? 0 : EPI_WARPS * 64 * 4);
  static constexpr int BYTES = END + 1024;  // + alignment slack for the dynamic smem base
  static_assert(BYTES <= 227 * 1024, "shared memory per CTA");
};

// Bounded wait whose completion must also make remote (peer CTA) writes visible.
__device__ __forceinline__ bool mbar_try_wait_cluster(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{.reg .pred p; mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p;}"
      : "=r"(ok) : "r"(bar), "r"(parity) : "memory");
  return ok != 0;
}
__device__ __forceinline__ bool mbar_wait_cluster(uint32_t bar, uint32_t parity, const volatile int *abort_flag,
                                                  uint64_t limit_ns) {
  if (mbar_try_wait_cluster(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (;;) {
#pragma unroll 1
    for (int i = 0; i < 32; ++i)
      if (mbar_try_wait_cluster(bar, parity)) return true;
    if (*abort_flag) return false;
    if (globaltimer_ns() - t0 > limit_ns) return false;
  }
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  uint32_t r;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}

__device__ __forceinline__ float ex2_approx(float x) {
  float r;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}

// GELU(t) = t * Phi(t), Phi the standard normal CDF, as max(t, 0) - |t| h with h = Phi(-|t|) (t (1 - h)
// for t >= 0, t h for t < 0, no 1 - erf cancellation). h = 2^P(x), x = min(|t|, 6), P the degree-10
// polynomial fitted to log2 Phi(-x) on [0, 6] (least squares on Chebyshev nodes, reweighted towards
// equal ripple): GELU within 4e-7 relative for |t| <= 0.1 and 2.5e-6 (float32 rounding included)
// elsewhere; at x = 6 the tail is below 1e-9, so clamping there costs less than 1e-9 |t|.
// Branch-free, one MUFU op (the erfc form with a reciprocal needs two, and MUFU throughput bounds
// the GELU epilogue).
__device__ __forceinline__ float gelu_erf(float t) {
  const float x = fminf(fabsf(t), 6.f);
  float p = -1.231680357705045e-08f;
  p = fmaf(p, x, 4.146599508203508e-07f);
  p = fmaf(p, x, -5.938332378718769e-06f);
  p = fmaf(p, x, 4.5272547140484676e-05f);
  p = fmaf(p, x, -0.0001642438000999391f);
  p = fmaf(p, x, -0.00026072203763760626f);
  p = fmaf(p, x, 0.007299995981156826f);
  p = fmaf(p, x, -0.05271168798208237f);
  p = fmaf(p, x, -0.45911723375320435f);
  p = fmaf(p, x, -1.151119351387024f);
  p = fmaf(p, x, -0.9999996423721313f);
  const float h = ex2_approx(p);
  return fmaf(-fabsf(t), h, fmaxf(t, 0.f));
}

// Two float32 lanes in one 64-bit register: fma / add of pairs (sm_100+ packed fp32 arithmetic,
// each lane the IEEE float32 operation, so results equal the scalar ones).
__device__ __forceinline__ uint64_t pk2(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void unpk2(uint64_t v, float &lo, float &hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t fma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
  return r;
}
__device__ __forceinline__ uint64_t add2(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__host__ __device__ constexpr uint64_t splat2(uint32_t bits) { return ((uint64_t)bits << 32) | bits; }

// gelu_erf of two values at once: the polynomial in packed pairs (half the FMA instructions).
__device__ __forceinline__ void gelu_erf2(float &a, float &b) {
  const uint64_t x = pk2(fminf(fabsf(a), 6.f), fminf(fabsf(b), 6.f));
  uint64_t p = splat2(__float_as_uint(-1.231680357705045e-08f));
  p = fma2(p, x, splat2(__float_as_uint(4.146599508203508e-07f)));
  p = fma2(p, x, splat2(__float_as_uint(-5.938332378718769e-06f)));
  p = fma2(p, x, splat2(__float_as_uint(4.5272547140484676e-05f)));
  p = fma2(p, x, splat2(__float_as_uint(-0.0001642438000999391f)));
  p = fma2(p, x, splat2(__float_as_uint(-0.00026072203763760626f)));
  p = fma2(p, x, splat2(__float_as_uint(0.007299995981156826f)));
  p = fma2(p, x, splat2(__float_as_uint(-0.05271168798208237f)));
  p = fma2(p, x, splat2(__float_as_uint(-0.45911723375320435f)));
  p = fma2(p, x, splat2(__float_as_uint(-1.151119351387024f)));
  p = fma2(p, x, splat2(__float_as_uint(-0.9999996423721313f)));
  float pa, pb;
  unpk2(p, pa, pb);
  const uint64_t h = pk2(ex2_approx(pa), ex2_approx(pb));
  const uint64_t r = fma2(pk2(-fabsf(a), -fabsf(b)), h, pk2(fmaxf(a, 0.f), fmaxf(b, 0.f)));
  unpk2(r, a, b);
}

// mbarrier arrival without release semantics: for signals that hand over no memory written by this
// thread (a TMEM buffer whose loads have completed, see tcgen05.wait::ld), so that the arrival does
// not wait for this thread's outstanding global stores.
__device__ __forceinline__ void mbar_arrive_relaxed(uint32_t bar) {
  asm volatile("mbarrier.arrive.relaxed.cta.shared::cta.b64 _, [%0];" :: "r"(bar) : "memory");
}
__device__ __forceinline__ void mbar_arrive_relaxed_cluster(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.relaxed.cluster.shared::cluster.b64 _, [%0];" :: "r"(cluster_addr) : "memory");
}

// Chain counters: a gpu-scope release increment (cumulative: it publishes the stores that this thread
// has acquired, i.e. those of every epilogue warp of the CTA) and its acquiring, bounded wait.
__device__ __forceinline__ void red_release_gpu_add(uint32_t *p, uint32_t v) {
  asm volatile("red.release.gpu.global.add.u32 [%0], %1;" :: "l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ uint32_t ld_acquire_gpu(const uint32_t *p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
// Warp-collective: true once every lane has read a count >= need (each lane's own acquire); false
// after limit_ns or once the CTA's abort flag is up.
__device__ __forceinline__ bool wait_count(const uint32_t *p, uint32_t need, const volatile int *abort_flag,
                                           uint64_t limit_ns) {
  if (__all_sync(0xffffffffu, ld_acquire_gpu(p) >= need)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (;;) {
    __nanosleep(128);
    if (__all_sync(0xffffffffu, ld_acquire_gpu(p) >= need)) return true;
    if (__any_sync(0xffffffffu, *abort_flag != 0)) return false;
    if (__any_sync(0xffffffffu, globaltimer_ns() - t0 > limit_ns)) return false;
  }
}

__device__ __forceinline__ void st_global_32B(void *p, const uint32_t (&w)[8]) {
  asm volatile("st.global.L1::no_allocate.v8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"l"(p), "r"(w[0]), "r"(w[1]), "r"(w[2]),
               "r"(w[3]), "r"(w[4]), "r"(w[5]), "r"(w[6]), "r"(w[7])
               : "memory");
}
__device__ __forceinline__ void ld_global_32B(const void *p, uint32_t (&w)[8]) {
  asm volatile("ld.global.v8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
               : "=r"(w[0]), "=r"(w[1]), "=r"(w[2]), "=r"(w[3]), "=r"(w[4]), "=r"(w[5]), "=r"(w[6]), "=r"(w[7])
               : "l"(p));
}

// Entry g of a table spread over the warp (lane l holds entries l + 32 j in t[j]); g warp-uniform.
template <int N>
__device__ __forceinline__ int table_at(const int (&t)[N], int g) {
  int v = 0;
#pragma unroll
  for (int j = 0; j < N; ++j) {
    const int x = __shfl_sync(0xffffffffu, t[j], g & 31);
    v = (g >> 5) == j ? x : v;
  }
  return v;
}

// The outputs of one run of 16 consecutive group rows (features f0 .. f0 + 15) for the lane's token
// t: y[0..16) are its accumulated sums (or zero), bs the run's bias in shared memory (the same for
// every lane). Adds the bias, applies GELU, rounds and stores the lane's 32-byte (bf16) or 64-byte
// (fp32) row segment with 32-byte stores, so that each store instruction writes whole sectors;
// bf16 output may add the residual (each sum rounded, as a separate bf16 addition would). GELU
// compiles the activation in; do_gelu applies it (a chain decides per linear).
template <bool GELU, bool F32, bool BIASG>
__device__ __forceinline__ void emit_run16(float (&y)[16], uint32_t bs, int f0, int64_t t, const LinearParams &P,
                                           bool do_gelu) {
#pragma unroll
  for (int i = 0; i < 16; i += 4) {
    uint64_t b01 = 0, b23 = 0;
    if (!BIASG) {
      asm volatile("ld.shared.v2.b64 {%0, %1}, [%2];" : "=l"(b01), "=l"(b23) : "r"(bs + 4 * i));
    } else if (P.bias != nullptr) {  // the same 16 features for every lane: a broadcast load from L1
      float4 bb;
      if (P.bias_vec16) {
        bb = __ldg(reinterpret_cast<const float4 *>(P.bias + f0 + i));
      } else {
        bb = make_float4(__ldg(P.bias + f0 + i), __ldg(P.bias + f0 + i + 1), __ldg(P.bias + f0 + i + 2),
                         __ldg(P.bias + f0 + i + 3));
      }
      b01 = pk2(bb.x, bb.y);
      b23 = pk2(bb.z, bb.w);
    }
    unpk2(add2(pk2(y[i], y[i + 1]), b01), y[i], y[i + 1]);
    unpk2(add2(pk2(y[i + 2], y[i + 3]), b23), y[i + 2], y[i + 3]);
  }
  if (GELU && do_gelu) {
#pragma unroll
    for (int i = 0; i < 16; i += 2) gelu_erf2(y[i], y[i + 1]);
  }
  if (t >= P.m) return;
  if (F32) {
    float *dst = static_cast<float *>(P.Y) + t * P.ldy + f0;
    if (P.y_vec32) {
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        uint32_t w[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) w[q] = __float_as_uint(y[8 * h + q]);
        st_global_32B(dst + 8 * h, w);
      }
    } else if (P.y_vec16) {
#pragma unroll
      for (int q = 0; q < 4; ++q) reinterpret_cast<float4 *>(dst)[q] = make_float4(y[4 * q], y[4 * q + 1], y[4 * q + 2], y[4 * q + 3]);
    } else {  // row not 16-byte aligned: element by element
#pragma unroll
      for (int q = 0; q < 16; ++q) dst[q] = y[q];
    }
  } else {
    uint32_t o[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) o[i] = pack_bf16x2(y[2 * i], y[2 * i + 1]);
    if (P.R != nullptr) {
      // a plain load: R may be Y itself, read and then written by this lane only
      const uint16_t *src = P.R + t * P.ldr + f0;
      uint32_t rw[8];
      if (P.r_vec32) {
        ld_global_32B(src, rw);
      } else {
        const int4 r0 = reinterpret_cast<const int4 *>(src)[0], r1 = reinterpret_cast<const int4 *>(src)[1];
        rw[0] = (uint32_t)r0.x; rw[1] = (uint32_t)r0.y; rw[2] = (uint32_t)r0.z; rw[3] = (uint32_t)r0.w;
        rw[4] = (uint32_t)r1.x; rw[5] = (uint32_t)r1.y; rw[6] = (uint32_t)r1.z; rw[7] = (uint32_t)r1.w;
      }
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        const float lo = __uint_as_float(o[q] << 16) + __uint_as_float(rw[q] << 16);
        const float hi = __uint_as_float(o[q] & 0xffff0000u) + __uint_as_float(rw[q] & 0xffff0000u);
        o[q] = pack_bf16x2(lo, hi);
      }
    }
    uint16_t *dst = static_cast<uint16_t *>(P.Y) + t * P.ldy + f0;
    if (P.y_vec32) {
      st_global_32B(dst, o);
    } else if (P.y_vec16) {
      reinterpret_cast<int4 *>(dst)[0] = make_int4((int)o[0], (int)o[1], (int)o[2], (int)o[3]);
      reinterpret_cast<int4 *>(dst)[1] = make_int4((int)o[4], (int)o[5], (int)o[6], (int)o[7]);
    } else {  // row not 16-byte aligned: element by element
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        dst[2 * q] = (uint16_t)(o[q] & 0xffffu);
        dst[2 * q + 1] = (uint16_t)(o[q] >> 16);
      }
    }
  }
}

// The pair kernel. One linear: tensor maps tmX0 / tmW0 and parameters P, C unused. A chain (CHAIN):
// C the launch's table, P its first linear's parameters (workspace, token count, timeout), GELU
// compiled in and applied to the linears that ask for it.
template <bool GELU, bool F32, bool DEEP, bool CHAIN>
__device__ __forceinline__ void pair_body(const CUtensorMap *tmX0, const CUtensorMap *tmW0, const LinearParams &P,
                                          const ChainParams *C) {
  using L = Smem<DEEP>;
  constexpr int NSTAGES = L::NSTAGES;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t smem_base = smem_u32(smem);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t rank = cluster_rank();  // 0: the pair's leader (schedules, issues the MMAs), 1: its peer
  const bool leader = rank == 0;

  const uint32_t bar0 = smem_base + L::BAR_OFF;
  auto full_bar = [&](int i) { return bar0 + 8u * i; };
  auto empty_bar = [&](int i) { return bar0 + 8u * (NSTAGES + i); };
  constexpr int RB = 2 * NSTAGES;  // first barrier after the stage ring
  auto accf_bar = [&](int b) { return bar0 + 8u * (RB + b); };
  auto acce_bar = [&](int b) { return bar0 + 8u * (RB + 2 + b); };
  auto unitf_bar = [&](int u) { return bar0 + 8u * (RB + 4 + u); };
  auto unite_bar = [&](int u) { return bar0 + 8u * (RB + 4 + UR + u); };
  const uint32_t drain_bar = bar0 + 8u * (RB + 4 + 2 * UR);
  auto stored_bar = [&](int b) { return bar0 + 8u * (RB + 5 + 2 * UR + b); };  // chain: a unit's stores
  UnitSlot *ring = reinterpret_cast<UnitSlot *>(smem + L::RING_OFF);
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + L::MISC_OFF);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(smem + L::MISC_OFF + 4);
  volatile int *never_flag = reinterpret_cast<volatile int *>(smem + L::MISC_OFF + 8);  // stays 0
  volatile int *chain_ok_s = reinterpret_cast<volatile int *>(smem + L::MISC_OFF + 12);  // chain: plans checked
  volatile int *last_cta_s = reinterpret_cast<volatile int *>(smem + L::MISC_OFF + 16);  // chain: last CTA out
  // the parameters of the unit's linear (a chain's record names it; one linear: P)
  auto jobp = [&](int j) -> const LinearParams & {
    if constexpr (CHAIN) return C->job[j].P;
    else return P;
  };

  const int32_t *gent = P.sched + SCHED_HDR_INTS;
  const int32_t *gpan = P.sched + sched_gpan_offset_ints(P.n_groups);
  const int32_t *entries = P.sched + sched_entries_offset_ints(P.n_groups);
  const int kc = sched_chunks(P.k);
  const uint64_t tmo = P.timeout_ns;

  // ---------------------------------------------------------------- prologue
  if (warp == 1) {
    tmem_alloc_pair(smem_u32(tmem_slot), 512);  // one warp of each CTA, together
    tmem_relinquish_pair();
  }
  if (warp == 0) {  // the barriers initialised by the lanes of one warp, one or two each
    if (lane < NSTAGES) {
      mbar_init(full_bar(lane), 1);
      mbar_init(empty_bar(lane), 1);
    }
    if (lane < 2) {
      mbar_init(accf_bar(lane), 1);
      mbar_init(acce_bar(lane), 2 * EPI_WARPS);
      if (CHAIN) mbar_init(stored_bar(lane), EPI_WARPS);
    }
    if (lane < UR) {
      mbar_init(unitf_bar(lane), 1);
      mbar_init(unite_bar(lane), UNIT_CONSUMERS);
    }
    if (lane == 0) {
      mbar_init(drain_bar, 1);
      *abort_flag = 0;
      *never_flag = 0;
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if constexpr (CHAIN) {
    if (warp == 0)
      for (int j = lane; j < C->njobs; j += 32) {
        prefetch_tensormap(&C->job[j].tmX);
        prefetch_tensormap(&C->job[j].tmW);
      }
  } else if (warp == 0 && lane == 0) {
    prefetch_tensormap(tmX0);
    prefetch_tensormap(tmW0);
  }
  // the work list must be this weight's plan: layout, group count, shape
  auto plan_ok = [](const LinearParams &Q) {
    return Q.sched[3] == 0 && Q.sched[1] == Q.n_groups && Q.sched[4] == Q.n && Q.sched[5] == Q.k &&
           Q.sched[6] == Q.bn && Q.sched[8] == SCHED_VERSION && Q.n_groups <= MAX_GROUPS;
  };
  bool sched_ok = !CHAIN && plan_ok(P);
  if constexpr (CHAIN) {
    if (warp == SCHED_WARP) {  // every linear's plan, a lane per linear (1 ok, 2 overflowed, 0 bad)
      bool ok = true, ovf = false;
      for (int j = lane; j < C->njobs; j += 32) {
        ok = ok && plan_ok(C->job[j].P);
        ovf = ovf || C->job[j].P.sched[3] != 0;
      }
      ok = __all_sync(0xffffffffu, ok);
      ovf = __any_sync(0xffffffffu, ovf);
      if (lane == 0) *chain_ok_s = ok ? 1 : (ovf ? 2 : 0);
    }
  }
  // When no group is cut into slices (S >= the chunk count), pair p's first unit is unit p: token
  // tile p / n_groups, group p % n_groups, all of that group's entries. The producers and the MMA
  // issuer take it from the work list themselves rather than wait for the scheduler's record (which
  // is the same); the group's entry range is requested here, so the load overlaps the prologue.
  const uint32_t u0 = blockIdx.x / 2;
  const uint32_t unsplit_units = (uint32_t)P.n_tt * (uint32_t)P.n_groups;
  const bool first_local = !CHAIN && sched_ok && P.S >= kc && (warp == 0 || warp == 1 || warp == W_WARP);
  int f_ga = 0, f_gb = 0;
  if (first_local && u0 < unsplit_units) {
    const int g = (int)(u0 % (uint32_t)P.n_groups);
    f_ga = __ldg(gent + g);
    f_gb = __ldg(gent + g + 1);
  }
  auto first_unit = [&](UnitInfo &d) {
    if (u0 < unsplit_units) {
      d.tt = (int)(u0 / (uint32_t)P.n_groups);
      d.g = (int)(u0 % (uint32_t)P.n_groups);
      d.s = 0;
      d.nsl = 1;
      d.e0 = f_ga;
      d.e1 = f_gb;
      d.ptile = (int)u0;
    } else {
      d.tt = -1; d.g = d.s = d.nsl = d.e0 = d.e1 = d.ptile = 0;
    }
    d.pad = 0;
  };
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // both CTAs' barriers are initialised before any signal crosses the pair
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  if constexpr (CHAIN) sched_ok = *chain_ok_s == 1;
  if (!sched_ok && tid == 0 && leader) {
    const bool ovf = CHAIN ? *chain_ok_s == 2 : P.sched[3] != 0;
    atomicOr(&P.ctl->err, ovf ? ERR_SCHED_OVERFLOW : ERR_BAD_SCHED);
  }

  if (warp == 0 || warp == W_WARP) {
    // ============================================================== producers
    const bool xrole = warp == 0;           // X tiles (else weight tiles)
    uint32_t it = 0, ui = 0;
    bool ok = true;
    while (ok) {
      const uint32_t slot = ui % UR, uph = (ui / UR) & 1u;
      UnitInfo inf;
      int cw;  // chunk indices of entries win .. win + 31, one per lane
      if (ui == 0 && first_local) {
        first_unit(inf);
        cw = inf.e0 + lane < inf.e1 ? __ldg(entries + inf.e0 + lane) : 0;
      } else {
        if (!mbar_wait_cluster(unitf_bar(slot), uph, abort_flag, tmo)) {
          ok = false;
          if (lane == 0) atomicOr(&P.ctl->err, ERR_PRODUCER_UNIT);
          break;
        }
        inf = ring[slot].inf;
        cw = ring[slot].win[lane];
      }
      __syncwarp();
      if (lane == 0) {
        if (leader) mbar_arrive(unite_bar(slot));
        else mbar_arrive_cluster(mapa_rank(unite_bar(slot), 0));
      }
      if (inf.tt < 0) break;
      const LinearParams &Q = jobp(inf.pad);
      const CUtensorMap *mX = tmX0, *mW = tmW0;
      const int32_t *ents = entries;
      int kcq = kc;
      if constexpr (CHAIN) {
        mX = &C->job[inf.pad].tmX;
        mW = &C->job[inf.pad].tmW;
        ents = Q.sched + sched_entries_offset_ints(Q.n_groups);
        kcq = sched_chunks(Q.k);
        if (xrole && inf.pad > 0 && inf.e1 > inf.e0) {
          // the previous linear's outputs of this token tile, all of them stored, before the copies
          const uint32_t need = 2u * (uint32_t)C->job[inf.pad - 1].P.n_groups;
          if (!wait_count(C->tile_done + (size_t)(inf.pad - 1) * C->n_tt + inf.tt, need, abort_flag, tmo)) {
            ok = false;
            if (lane == 0) atomicOr(&P.ctl->err, ERR_CHAIN_WAIT);
            break;
          }
          asm volatile("fence.proxy.async.global;" ::: "memory");  // order the tensor copies after the acquire
        }
      }
      // Stages: a batch of up to BATCH consecutive entries; lane i < nb waits for stage i's empty
      // barrier, then issues its stage's copy (this warp's kind), completing on the leader's full
      // barrier; the leader's X producer posts the stage's expected bytes (both kinds, both CTAs).
      const int ytok = inf.tt * TOKENS_PER_TILE + (int)rank * CTA_TOKENS;
      int win = inf.e0;
      int cw_next = xrole && win + 32 + lane < inf.e1 ? __ldg(ents + win + 32 + lane) : 0;
      for (int base = inf.e0; base < inf.e1 && ok; base += BATCH) {
        const int nb = min(BATCH, inf.e1 - base);
        if (base >= win + 32) {  // BATCH divides 32: a batch never straddles two windows
          win += 32;
          cw = cw_next;
          cw_next = xrole && win + 32 + lane < inf.e1 ? __ldg(ents + win + 32 + lane) : 0;
        }
        const int e = base + (lane < nb ? lane : 0);  // the batch entry of this lane's copy
        int c = __shfl_sync(0xffffffffu, cw, (e - win) & 31);
        int tile = e;
        // a chunk or tile outside the work list's ranges means a corrupt list: flag it, load tile 0
        const bool in_range = xrole ? (c >= 0 && c < kcq) : ((int64_t)tile < Q.stream_tiles);
        if (!in_range) {
          c = 0;
          tile = 0;
        }
        const uint32_t itk = it + (uint32_t)lane;
        const uint32_t stk = itk % NSTAGES;
        const uint32_t st = smem_base + stk * STAGE_BYTES;
        const uint32_t fb = mapa_rank(full_bar(stk), 0);
        bool wok = true;
        if (lane < nb) wok = mbar_wait(empty_bar(stk), ((itk / NSTAGES) & 1u) ^ 1u, abort_flag, tmo);
        if (!__all_sync(0xffffffffu, wok)) {
          ok = false;
          if (lane == 0) atomicOr(&P.ctl->err, ERR_PRODUCER_EMPTY);
          break;
        }
        if (lane < nb) {  // the batch's stages are all free: one issue step for all of them
          if (!in_range) atomicOr(&P.ctl->err, ERR_BAD_SCHED);
          if (leader && xrole) mbar_arrive_expect_tx(full_bar(stk), 2 * STAGE_BYTES);
          if (xrole) tma_load_2d_pair(st, mX, c * CHUNK_COLS, ytok, fb);
          else tma_load_2d_pair(st + X_BYTES, mW, 0, tile * GROUP_FEATURES + (int)rank * HALF_FEATURES, fb);
        }
        __syncwarp();
        it += nb;
      }
      if (!ok) break;
      ++ui;
    }
    if (!ok && lane == 0) *abort_flag = 1;
    // no copy of either CTA may still be in flight: they all complete on the leader's full barriers
    if (leader && xrole) {
      const uint32_t first = it > (uint32_t)NSTAGES ? it - NSTAGES : 0u;
      for (uint32_t i = first; i < it; ++i)
        if (!mbar_wait(full_bar(i % NSTAGES), (i / NSTAGES) & 1u, never_flag, tmo)) {
          if (lane == 0) atomicOr(&P.ctl->err, ERR_DRAIN);
          break;
        }
    }
  } else if (warp == SCHED_WARP) {
    // ============================================================== scheduler (leader only)
    // Publishes each unit (or the end record) once its ring slot is free in both CTAs: the record
    // and the unit's first 32 chunk indices, written locally and into the peer, then both CTAs'
    // unit-full barriers. Runs up to UR units ahead of the producers.
    if (leader) {
      bool ok = true, queued = false;
      // the first unit of pair p is unit p (no queue round trip before the first copies); the queue
      // hands out the units after the first gridDim.x / 2. When every unit is such a first unit
      // (small token counts), no pair touches the queue or its counters.
      const uint32_t npairs = gridDim.x / 2;
      uint32_t fetched = blockIdx.x / 2;
      // waits for ring slot `pub` to be free in both CTAs
      auto slot_free = [&](uint32_t pub) -> bool {
        if (mbar_wait_cluster(unite_bar(pub % UR), ((pub / UR) & 1u) ^ 1u, abort_flag, tmo)) return true;
        ok = false;
        if (lane == 0) atomicOr(&P.ctl->err, ERR_PRODUCER_UNIT);
        return false;
      };
      // writes record d and its first 32 chunk indices (from ents) into slot `pub` of both CTAs
      auto publish = [&](uint32_t pub, const UnitInfo &d, const int32_t *ents) {
        const uint32_t slot = pub % UR;
        const int wv = d.e0 + lane < d.e1 ? __ldg(ents + d.e0 + lane) : 0;
        UnitSlot &rs = ring[slot];
        const uint32_t remote = mapa_rank(smem_u32(&rs), 1);
        rs.win[lane] = wv;
        asm volatile("st.shared::cluster.b32 [%0], %1;"
                     :: "r"(remote + (uint32_t)offsetof(UnitSlot, win) + 4u * lane), "r"(wv) : "memory");
        if (lane == 0) {
          rs.inf = d;
          const int4 *v = reinterpret_cast<const int4 *>(&d);
          st_cluster_v4(remote, v[0]);
          st_cluster_v4(remote + 16, v[1]);
        }
        asm volatile("fence.acq_rel.cluster;" ::: "memory");  // every lane's writes before the signal
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(unitf_bar(slot));
          mbar_arrive_cluster(mapa_rank(unitf_bar(slot), 1));
        }
        __syncwarp();
      };
      if constexpr (CHAIN) {
        // units in order: linear 0's (token-tile-major), then linear 1's, ...; a unit never cut
        const uint32_t total_units = sched_ok ? C->total_units : 0u;
        queued = total_units > npairs;
        int jc = 0;  // the linear of the last unit taken (units come in increasing order)
        for (uint32_t pub = 0;; ++pub) {
          if (!slot_free(pub)) break;
          const uint32_t u = __shfl_sync(0xffffffffu, fetched, 0);
          UnitInfo d;
          const int32_t *ents = nullptr;
          if (u < total_units) {
            while (jc + 1 < C->njobs && u >= C->job[jc].unit0 + C->job[jc].units) ++jc;
            const LinearParams &Q = C->job[jc].P;
            const uint32_t r = u - C->job[jc].unit0;
            d.tt = (int)(r / (uint32_t)Q.n_groups);
            d.g = (int)(r % (uint32_t)Q.n_groups);
            d.s = 0;
            d.nsl = 1;
            d.e0 = __ldg(Q.sched + SCHED_HDR_INTS + d.g);
            d.e1 = __ldg(Q.sched + SCHED_HDR_INTS + d.g + 1);
            d.ptile = (int)r;
            d.pad = jc;
            ents = Q.sched + sched_entries_offset_ints(Q.n_groups);
          } else {
            d.tt = -1; d.g = d.s = d.nsl = d.e0 = d.e1 = d.ptile = d.pad = 0;
          }
          if (lane == 0 && u < total_units) fetched = queued ? npairs + atomicAdd(&P.ctl->next_unit, 1u) : total_units;
          publish(pub, d, ents);
          if (u >= total_units) break;
        }
      } else {
        // slices per group = max(1, ceil(entries / S)) and their exclusive prefix, kept in registers:
        // lane l holds group l + 32 j in sp[j] (first slice) and ge[j] (first entry)
        constexpr int GPL = MAX_GROUPS / 32;
        int sp[GPL], ge[GPL];
        int run = 0;
#pragma unroll
        for (int j = 0; j < GPL; ++j) {
          const int g = 32 * j + lane;
          int c = 0, g0 = 0;
          if (sched_ok && g < P.n_groups) {
            g0 = gent[g];
            const int cnt = gent[g + 1] - g0;
            c = cnt <= 0 ? 1 : (cnt + P.S - 1) / P.S;
          }
          int incl = c;
#pragma unroll
          for (int o = 1; o < 32; o <<= 1) {
            const int t = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += t;
          }
          sp[j] = run + incl - c;
          ge[j] = g0;
          run += __shfl_sync(0xffffffffu, incl, 31);
        }
        const int total_slices = run;
        const int ge_end = sched_ok ? gent[P.n_groups] : 0;
        const uint32_t total_units = sched_ok ? (uint32_t)P.n_tt * (uint32_t)total_slices : 0u;
        queued = total_units > npairs;  // the same in every pair
        for (uint32_t pub = 0;; ++pub) {
          if (!slot_free(pub)) break;
          const uint32_t u = __shfl_sync(0xffffffffu, fetched, 0);
          UnitInfo d;
          if (u < total_units) {
            d.tt = (int)(u / (uint32_t)total_slices);
            const int rr = (int)(u % (uint32_t)total_slices);
            // group g with sp[g] <= rr < sp[g + 1]: every group has a slice, so g + 1 = #{g : sp[g] <= rr}
            int cnt = 0;
#pragma unroll
            for (int j = 0; j < GPL; ++j)
              cnt += __popc(__ballot_sync(0xffffffffu, 32 * j + lane < P.n_groups && sp[j] <= rr));
            const int g = cnt - 1;
            const int s0 = table_at(sp, g), s1 = g + 1 < P.n_groups ? table_at(sp, g + 1) : total_slices;
            const int ge0 = table_at(ge, g), ge1 = g + 1 < P.n_groups ? table_at(ge, g + 1) : ge_end;
            d.g = g;
            d.s = rr - s0;
            d.nsl = s1 - s0;
            d.e0 = min(ge0 + d.s * P.S, ge1);
            d.e1 = min(d.e0 + P.S, ge1);
            d.ptile = d.tt * total_slices + rr;
          } else {
            d.tt = -1; d.g = d.s = d.nsl = d.e0 = d.e1 = d.ptile = 0;
          }
          d.pad = 0;
          if (lane == 0 && u < total_units) fetched = queued ? npairs + atomicAdd(&P.ctl->next_unit, 1u) : total_units;
          publish(pub, d, entries);
          if (u >= total_units) break;
        }
      }
      if (!ok && lane == 0) *abort_flag = 1;
      // queue bookkeeping: the last scheduler to leave resets the counters for the next launch
      if (lane == 0 && queued) {
        __threadfence();
        if (atomicAdd(&P.ctl->done_ctas, 1u) == gridDim.x / 2 - 1) {
          P.ctl->next_unit = 0;
          P.ctl->done_ctas = 0;
          __threadfence();
        }
      }
    }
  } else if (warp < FIRST_EPI) {
    // ============================================================== MMA issuer (leader only)
    if (leader) {
      uint32_t it = 0, ui = 0;
      bool ok = true;
      while (ok) {
        const uint32_t slot = ui % UR, uph = (ui / UR) & 1u;
        UnitInfo inf;
        if (ui == 0 && first_local) {
          first_unit(inf);
        } else {
          if (!mbar_wait(unitf_bar(slot), uph, abort_flag, tmo)) {
            ok = false;
            if (lane == 0) atomicOr(&P.ctl->err, ERR_MMA_UNIT);
            break;
          }
          inf = ring[slot].inf;
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(unite_bar(slot));
        if (inf.tt < 0) break;
        const uint32_t buf = ui & 1u, aph = (ui >> 1) & 1u;
        // both CTAs' epilogues have read this accumulator buffer
        if (!mbar_wait_cluster(acce_bar(buf), aph ^ 1u, abort_flag, tmo)) {
          ok = false;
          if (lane == 0) atomicOr(&P.ctl->err, ERR_MMA_ACC);
          break;
        }
        tc_fence_after();
        const uint32_t dbase = tmem_base + buf * BUF_COLS;
        for (int e = inf.e0; e < inf.e1; ++e) {
          const uint32_t stage = it % NSTAGES, ph = (it / NSTAGES) & 1u;
          if (!mbar_wait(full_bar(stage), ph, abort_flag, tmo)) {
            ok = false;
            if (lane == 0) atomicOr(&P.ctl->err, ERR_MMA_FULL);
            break;
          }
          tc_fence_after();
          const uint32_t st = smem_base + stage * STAGE_BYTES;
          if (elect_one()) {
#pragma unroll
            for (int kk = 0; kk < KSTEPS; ++kk) {
              const uint64_t adesc = smem_desc<128>(st + kk * 32);
              const uint64_t bdesc = smem_desc<128>(st + X_BYTES + kk * 32);
              umma_f16_pair(dbase, adesc, bdesc, IDESC, (e > inf.e0 || kk > 0) ? 1u : 0u);
            }
            tc_commit_pair(empty_bar(stage), 3);
          }
          __syncwarp();
          ++it;
        }
        if (!ok) break;
        if (elect_one()) {
          if (inf.e1 > inf.e0) {
            tc_commit_pair(accf_bar(buf), 3);
          } else {  // nothing accumulated: the epilogue treats the sums as zero
            mbar_arrive(accf_bar(buf));
            mbar_arrive_cluster(mapa_rank(accf_bar(buf), 1));
          }
        }
        __syncwarp();
        ++ui;
      }
      if (!ok && lane == 0) *abort_flag = 1;
      // every MMA this thread issued completes before TMEM can be freed
      if (elect_one()) tc_commit_pair(drain_bar, 1);
      __syncwarp();
      if (!mbar_wait(drain_bar, 0, never_flag, tmo) && lane == 0) atomicOr(&P.ctl->err, ERR_DRAIN);
    }
  } else {
    // ============================================================== epilogue
    // The accumulator is 128 tokens (TMEM lanes) x 256 group rows (columns). Warp w reads lane
    // quarter q = w % 4 (tokens 32 q .. 32 q + 31) and the 64 columns of part (w - 2) / 4.
    const int q = warp & 3;
    const int part = (warp - FIRST_EPI) >> 2;
    float *bias_s = reinterpret_cast<float *>(smem + L::BIAS_OFF) + (warp - FIRST_EPI) * 64;  // (not DEEP)
    // Takes the record of unit u and hands its ring slot back. The hand-back orders nothing but
    // this warp's reads of the slot, so it is a relaxed arrival made data-dependent on them: a vote
    // over every lane's loaded record (pad is always 0) completes only once all the reads have
    // returned. A release arrival would also wait for the previous unit's output stores.
    auto take_unit = [&](uint32_t u, UnitInfo &out) -> bool {
      const uint32_t slot = u % UR, uph = (u / UR) & 1u;
      if (!(leader ? mbar_wait(unitf_bar(slot), uph, abort_flag, tmo)
                   : mbar_wait_cluster(unitf_bar(slot), uph, abort_flag, tmo))) {
        if (lane == 0) { atomicOr(&P.ctl->err, ERR_EPI_UNIT); *abort_flag = 1; }
        return false;
      }
      out = ring[slot].inf;
      const uint32_t read = __ballot_sync(0xffffffffu, (out.tt ^ out.g ^ out.s ^ out.nsl ^ out.e0 ^ out.e1 ^ out.ptile) !=
                                                           0x7fffffff || out.pad >= 0);
      if (lane == 0 && read != 0u) {
        if (leader) mbar_arrive_relaxed(unite_bar(slot));
        else mbar_arrive_relaxed_cluster(mapa_rank(unite_bar(slot), 0));
      }
      return true;
    };
    UnitInfo inf;
    bool have = take_unit(0, inf);
    uint32_t ui = 0;
    while (have && inf.tt >= 0) {
      const LinearParams &Q = jobp(inf.pad);
      const int32_t *gp = CHAIN ? Q.sched + sched_gpan_offset_ints(Q.n_groups) : gpan;
      // the features of this warp's 64 columns (first feature of each 16-column quarter, or -1)
      int fcol[4];
#pragma unroll
      for (int r4 = 0; r4 < 4; ++r4) {
        const int c = 64 * part + 16 * r4;
        const int panel = __ldg(gp + (int64_t)inf.g * MAX_GROUP_PANELS + c / Q.bn);
        fcol[r4] = panel >= 0 ? panel * Q.bn + c % Q.bn : -1;
      }
      // and their bias, staged while the accumulator is still being computed
      if (!DEEP && lane < 16) {
        const int qq = lane >> 2;  // the lane's quarter, selected without indexing the array
        const int fq = qq == 0 ? fcol[0] : (qq == 1 ? fcol[1] : (qq == 2 ? fcol[2] : fcol[3]));
        const int f = fq < 0 ? -1 : fq + 4 * (lane & 3);
        float4 b4 = make_float4(0.f, 0.f, 0.f, 0.f);
        if (f >= 0 && Q.bias != nullptr) {
          if (Q.bias_vec16) {
            b4 = __ldg(reinterpret_cast<const float4 *>(Q.bias + f));
          } else {
            b4 = make_float4(__ldg(Q.bias + f), __ldg(Q.bias + f + 1), __ldg(Q.bias + f + 2), __ldg(Q.bias + f + 3));
          }
        }
        *reinterpret_cast<float4 *>(bias_s + 4 * lane) = b4;
      }
      __syncwarp();
      const uint32_t buf = ui & 1u, aph = (ui >> 1) & 1u;
      if (!mbar_wait(accf_bar(buf), aph, abort_flag, tmo)) {
        if (lane == 0) { atomicOr(&P.ctl->err, ERR_EPI_ACC); *abort_flag = 1; }
        break;
      }
      tc_fence_after();
      const int t_tile = (int)rank * CTA_TOKENS + 32 * q + lane;   // token within the unit's tile
      const int64_t tok0 = (int64_t)inf.tt * TOKENS_PER_TILE + (int)rank * CTA_TOKENS + 32 * q;
      const int64_t t = tok0 + lane;
      const bool tvalid = t < P.m;
      const bool split = inf.nsl > 1;
      const bool touched = inf.e1 > inf.e0;
      if constexpr (CHAIN) {
        // a unit with no entries loads nothing, so no copy waited for the previous linear: its
        // stores wait here, so that they follow every earlier linear's use of this token tile
        if (!touched && inf.pad > 0 &&
            !wait_count(C->tile_done + (size_t)(inf.pad - 1) * C->n_tt + inf.tt,
                        2u * (uint32_t)C->job[inf.pad - 1].P.n_groups, abort_flag, tmo)) {
          if (lane == 0) { atomicOr(&P.ctl->err, ERR_CHAIN_WAIT); *abort_flag = 1; }
          break;
        }
      }
      const bool do_gelu = !CHAIN || Q.gelu != 0;
      float *part_row = nullptr;
      if (split)
        part_row = P.partials + ((int64_t)inf.ptile * P.part_rows + t_tile) * GROUP_FEATURES;
      // the next unit's record, before this unit's stores
      UnitInfo nxt;
      have = take_unit(ui + 1, nxt);
#pragma unroll 1
      for (int h = 0; h < 2; ++h) {
        const int c0 = 64 * part + 32 * h;  // first group row (accumulator column) of these 32
        float v[32];
        if (touched) {  // warp-uniform: the TMEM load is a warp-collective instruction
          tmem_ld32(tmem_base + ((uint32_t)(32 * q) << 16) + buf * BUF_COLS + c0, v);
        } else {
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] = 0.f;
        }
        if (split) {
          if (tvalid) {
            float4 *dst = reinterpret_cast<float4 *>(part_row + c0);
#pragma unroll
            for (int i = 0; i < 8; ++i) dst[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
          }
        } else {
          const int fa = h == 0 ? fcol[0] : fcol[2], fb2 = h == 0 ? fcol[1] : fcol[3];
          float ya[16], yb[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            ya[i] = v[i];
            yb[i] = v[16 + i];
          }
          const uint32_t bs = smem_u32(bias_s + 32 * h);
          if (fa >= 0) emit_run16<GELU, F32, DEEP>(ya, bs, fa, t, Q, do_gelu);
          if (fb2 >= 0) emit_run16<GELU, F32, DEEP>(yb, bs + 64, fb2, t, Q, do_gelu);
        }
        __syncwarp();
      }
      if constexpr (CHAIN) {
        // this warp's stores of the unit are done (a CTA-scope release); arriving before the
        // accumulator hand-back means a stored barrier phase always completes before the MMAs of
        // the unit two ahead, which reuses it, can start
        __syncwarp();
        if (lane == 0) mbar_arrive(stored_bar((int)(ui & 1u)));
      }
      // the accumulator buffer is free again (the leader's MMAs wait for both CTAs' warps); its
      // loads have completed and no memory written here is handed over, so no release ordering
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (leader) mbar_arrive_relaxed(acce_bar(buf));
        else mbar_arrive_relaxed_cluster(mapa_rank(acce_bar(buf), 0));
      }
      if constexpr (CHAIN) {
        // one epilogue warp per unit, in turn, publishes the CTA's stores of it to the next linear:
        // it acquires the 16 warps' arrivals, then counts them with a gpu-scope release (which waits
        // for the stores to complete; taking turns spreads that wait over the warps)
        if (warp == FIRST_EPI + (int)(ui % (uint32_t)EPI_WARPS)) {
          if (!mbar_wait(stored_bar((int)(ui & 1u)), (ui >> 1) & 1u, abort_flag, tmo)) {
            if (lane == 0) { atomicOr(&P.ctl->err, ERR_CHAIN_WAIT); *abort_flag = 1; }
            break;
          }
          if (lane == 0) red_release_gpu_add(C->tile_done + (size_t)inf.pad * C->n_tt + inf.tt, 1u);
        }
      }
      inf = nxt;
      ++ui;
    }
  }

  // ---------------------------------------------------------------- teardown
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // no signal, copy or MMA of the pair is still aimed at either CTA
  tc_fence_after();
  if (warp == 1) tmem_dealloc_pair(tmem_base, 512);
  if constexpr (CHAIN) {
    // the last CTA out (every other CTA has finished its waits and counts) clears the tile
    // counters for the next chain launch on this workspace
    if (tid == 0) {
      __threadfence();
      *last_cta_s = atomicAdd(&P.ctl->chain_ctas, 1u) == gridDim.x - 1 ? 1 : 0;
    }
    __syncthreads();
    if (*last_cta_s) {
      __threadfence();
      const int count = C->njobs * C->n_tt;
      for (int i = tid; i < count; i += NUM_THREADS) C->tile_done[i] = 0u;
      if (tid == 0) P.ctl->chain_ctas = 0u;
      __threadfence();
    }
  }
}

template <bool GELU, bool F32, bool DEEP>
__global__ void __launch_bounds__(NUM_THREADS, 1)
bsr_linear_kernel(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmW,
                  const LinearParams P) {
  pair_body<GELU, F32, DEEP, false>(&tmX, &tmW, P, nullptr);
}

// Chains: bf16 outputs, six stages with the staged bias (the long-K linears lose their seventh
// stage), GELU per linear.
__global__ void __launch_bounds__(NUM_THREADS, 1) bsr_linear_chain_kernel(const __grid_constant__ ChainParams C) {
  pair_body<true, false, false, true>(nullptr, nullptr, C.job[0].P, &C);
}

// Split units: Y = act(sum over the slices, in slice order, of the partial sums + bias). One thread
// per 8 consecutive group rows of one token of one (token tile, group) with more than one slice.
__global__ void __launch_bounds__(256) split_reduce_kernel(const ReduceParams R) {
  __shared__ int sp[MAX_GROUPS + 1];
  __shared__ int nslice[MAX_GROUPS];
  const int32_t *gent = R.sched + SCHED_HDR_INTS;
  const int32_t *gpan = R.sched + sched_gpan_offset_ints(R.n_groups);
  if (threadIdx.x < 32) {
    int run = 0;
    const int lane = threadIdx.x;
    for (int base = 0; base < R.n_groups; base += 32) {
      const int g = base + lane;
      int c = 0;
      if (g < R.n_groups) {
        const int cnt = gent[g + 1] - gent[g];
        c = cnt <= 0 ? 1 : (cnt + R.S - 1) / R.S;
        nslice[g] = c;
      }
      int incl = c;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int tv = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += tv;
      }
      if (g < R.n_groups) sp[g] = run + incl - c;
      run += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (lane == 0) sp[R.n_groups] = run;
  }
  __syncthreads();
  const int total_slices = sp[R.n_groups];
  constexpr int VPR = GROUP_FEATURES / 8;  // 8-row pieces per token
  const int64_t items = (int64_t)R.n_tt * R.n_groups * R.part_rows * VPR;
  for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < items; idx += (int64_t)gridDim.x * blockDim.x) {
    const int v = (int)(idx % VPR);
    int64_t rest = idx / VPR;
    const int row = (int)(rest % R.part_rows);
    rest /= R.part_rows;
    const int g = (int)(rest % R.n_groups);
    const int tt = (int)(rest / R.n_groups);
    const int nsl = nslice[g];
    if (nsl <= 1) continue;
    const int64_t t = (int64_t)tt * TOKENS_PER_TILE + row;
    if (t >= R.m) continue;
    const int c0 = 8 * v;
    const int panel = gpan[(int64_t)g * MAX_GROUP_PANELS + c0 / R.bn];
    if (panel < 0) continue;
    float acc[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) acc[i] = 0.f;
    const float *p0 = R.partials + (((int64_t)tt * total_slices + sp[g]) * R.part_rows + row) * GROUP_FEATURES + c0;
    for (int s = 0; s < nsl; ++s) {
      const float4 *p = reinterpret_cast<const float4 *>(p0 + (int64_t)s * R.part_rows * GROUP_FEATURES);
      const float4 a = __ldcg(p), b = __ldcg(p + 1);
      acc[0] += a.x; acc[1] += a.y; acc[2] += a.z; acc[3] += a.w;
      acc[4] += b.x; acc[5] += b.y; acc[6] += b.z; acc[7] += b.w;
    }
    {
      const int f0 = panel * R.bn + c0 % R.bn;
      float b8[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) b8[i] = R.bias != nullptr ? R.bias[f0 + i] : 0.f;
#pragma unroll
      for (int i = 0; i < 8; ++i) acc[i] = R.gelu ? gelu_erf(acc[i] + b8[i]) : acc[i] + b8[i];
      if (R.y_f32) {
        float *dst = static_cast<float *>(R.Y) + t * R.ldy + f0;
#pragma unroll
        for (int i = 0; i < 8; ++i) dst[i] = acc[i];
      } else {
        uint16_t *dst = static_cast<uint16_t *>(R.Y) + t * R.ldy + f0;
#pragma unroll
        for (int i = 0; i < 8; i += 2) {
          uint32_t w = pack_bf16x2(acc[i], acc[i + 1]);
          if (R.R != nullptr) {
            const uint16_t *rp = R.R + t * R.ldr + f0;
            const float lo = __uint_as_float(w << 16) + __uint_as_float((uint32_t)rp[i] << 16);
            const float hi = __uint_as_float(w & 0xffff0000u) + __uint_as_float((uint32_t)rp[i + 1] << 16);
            w = pack_bf16x2(lo, hi);
          }
          dst[i] = (uint16_t)(w & 0xffffu);
          dst[i + 1] = (uint16_t)(w >> 16);
        }
      }
    }
  }
}

// ------------------------------------------------------------------------------------ small m
// Token counts up to SMALL_M_MAX (batch 1 of a ViT is 197 tokens): the pair kernel's fixed cost --
// cluster launch, TMEM allocation for 512 columns, the scheduler's dependent loads, a second launch
// for split slices -- is most of such a call. Here plain CTAs of four warps each compute 128 tokens x
// 32 group rows of one group over a share of the group's entries, from the same work list and
// weight stream. All 128 threads copy each entry's X and weight rows with 16-byte cp.async into a
// five-stage ring (two CTAs per SM), in the 128-byte-swizzled K-major layout the tensor core reads (piece j of row r
// at j ^ (r mod 8) inside 1024-byte atoms); one thread issues the entry's four tcgen05 MMAs
// (M = 128 tokens, N = 32 rows, K = 16) into 32 TMEM columns and commits them to the stage's
// mbarrier, which frees the stage for its next copy. A long K is cut into kp parts run by the kp
// CTAs of one cluster; their partial sums meet in distributed shared memory and are added in rank
// order (deterministic), each CTA finishing 128 / kp of the tokens.
constexpr int SM_TOK = 128;                           // tokens per CTA: the MMA's M (a lane each)
constexpr int SM_ROWS = 32;                           // group rows per CTA: the MMA's N
constexpr int SM_SLICES = GROUP_FEATURES / SM_ROWS;   // row slices per group
constexpr int SM_THREADS = 128;
constexpr int SM_STAGES = 5;
constexpr int SM_XB = SM_TOK * CHUNK_COLS * 2;        // 16 KB of X per stage
constexpr int SM_WB = SM_ROWS * CHUNK_COLS * 2;       // 4 KB of the weight stream per stage
constexpr int SM_STAGE = SM_XB + SM_WB;
constexpr int SM_PSTRIDE = SM_ROWS + 4;               // floats per token row of the partial tile
constexpr int SM_CHUNK_OFF = SM_STAGES * SM_STAGE;    // then the CTA's chunk indices (kc ints)
constexpr uint32_t SM_IDESC = idesc_bf16(SM_TOK, SM_ROWS);
static_assert(SM_STAGE % 1024 == 0 && SM_XB % 1024 == 0, "stages and their weight rows start on swizzle atoms");
static_assert(SM_TOK * SM_PSTRIDE * 4 <= SM_STAGES * SM_STAGE, "the partial tile reuses the ring");

__device__ __forceinline__ float4 ld_cluster_f4(uint32_t addr) {
  float4 v;
  asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];" : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w) : "r"(addr));
  return v;
}

// Bias, GELU, rounding, residual and store of 8 consecutive features f0 .. f0 + 7 of token t (the
// same operations, in the same order, as the pair kernel's epilogue).
template <bool GELU, bool F32>
__device__ __forceinline__ void finish8(float *v, const float *b8, int f0, int64_t t, const LinearParams &P) {
  if (P.bias != nullptr) {
#pragma unroll
    for (int i = 0; i < 8; ++i) v[i] += b8[i];
  }
  if (GELU) {
#pragma unroll
    for (int i = 0; i < 8; i += 2) gelu_erf2(v[i], v[i + 1]);
  }
  if (F32) {
    float *dst = static_cast<float *>(P.Y) + t * P.ldy + f0;
    if (P.y_vec16) {
      reinterpret_cast<float4 *>(dst)[0] = make_float4(v[0], v[1], v[2], v[3]);
      reinterpret_cast<float4 *>(dst)[1] = make_float4(v[4], v[5], v[6], v[7]);
    } else {
#pragma unroll
      for (int i = 0; i < 8; ++i) dst[i] = v[i];
    }
  } else {
    uint32_t o[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) o[i] = pack_bf16x2(v[2 * i], v[2 * i + 1]);
    if (P.R != nullptr) {  // 16-byte rows (checked on the host); R may be Y itself, read before written
      const int4 r4 = *reinterpret_cast<const int4 *>(P.R + t * P.ldr + f0);
      const uint32_t rw[4] = {(uint32_t)r4.x, (uint32_t)r4.y, (uint32_t)r4.z, (uint32_t)r4.w};
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float lo = __uint_as_float(o[q] << 16) + __uint_as_float(rw[q] << 16);
        const float hi = __uint_as_float(o[q] & 0xffff0000u) + __uint_as_float(rw[q] & 0xffff0000u);
        o[q] = pack_bf16x2(lo, hi);
      }
    }
    uint16_t *dst = static_cast<uint16_t *>(P.Y) + t * P.ldy + f0;
    if (P.y_vec16) {
      *reinterpret_cast<int4 *>(dst) = make_int4((int)o[0], (int)o[1], (int)o[2], (int)o[3]);
    } else {
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        dst[2 * q] = (uint16_t)(o[q] & 0xffffu);
        dst[2 * q + 1] = (uint16_t)(o[q] >> 16);
      }
    }
  }
}

// Grid: kp x SM_SLICES x n_groups x ceil(m / SM_TOK) CTAs, clusters of kp along x.
template <bool GELU, bool F32>
__global__ void __launch_bounds__(SM_THREADS) bsr_linear_small_kernel(const LinearParams P) {
  extern __shared__ uint8_t sm_raw[];
  uint8_t *sm = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(sm_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t mma_bar[SM_STAGES];
  __shared__ __align__(16) float bias_s[SM_ROWS];  // the slice's bias (0 where the row has no panel)
  __shared__ uint32_t tmem_slot;
  __shared__ int abort_flag;  // stays 0: the waits end only by completion or their time limit
  const uint32_t ring = smem_u32(sm);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int kp = P.kp;
  const int part = (int)(blockIdx.x % (unsigned)kp);  // the cluster rank (clusters of kp along x)
  int idx = (int)(blockIdx.x / (unsigned)kp);
  const int rs = idx % SM_SLICES;
  idx /= SM_SLICES;
  const int g = idx % P.n_groups;
  const int tt = idx / P.n_groups;
  const int kc = sched_chunks(P.k);
  // one wave of independent loads: the header words, the group's entry range, this slice's panels
  // (one or two slots); every early return below depends only on data shared by the whole cluster
  const int32_t *gpan = P.sched + sched_gpan_offset_ints(P.n_groups) + (int64_t)g * MAX_GROUP_PANELS;
  const int32_t *gent = P.sched + SCHED_HDR_INTS;
  const int slot0 = rs * SM_ROWS / P.bn, slot1 = (rs * SM_ROWS + SM_ROWS - 1) / P.bn;
  const int h1 = __ldg(P.sched + 1), h3 = __ldg(P.sched + 3), h4 = __ldg(P.sched + 4), h5 = __ldg(P.sched + 5);
  const int h6 = __ldg(P.sched + 6), h8 = __ldg(P.sched + 8);
  const int ga = __ldg(gent + g), gb = __ldg(gent + g + 1);
  const int p0 = __ldg(gpan + slot0), p1 = __ldg(gpan + slot1);
  const bool sched_ok = h3 == 0 && h1 == P.n_groups && h4 == P.n && h5 == P.k && h6 == P.bn && h8 == SCHED_VERSION;
  if (!sched_ok) {
    if (blockIdx.x == 0 && tid == 0) atomicOr(&P.ctl->err, h3 ? ERR_SCHED_OVERFLOW : ERR_BAD_SCHED);
    return;
  }
  if (p0 < 0 && p1 < 0) return;  // a row slice with no panel (the last group of an n that is not a multiple of 256)
  if (ga < 0 || gb < ga || gb - ga > kc || (int64_t)gb > P.stream_tiles) {
    if (part == 0 && rs == 0 && tt == 0 && tid == 0) atomicOr(&P.ctl->err, ERR_BAD_SCHED);
    return;
  }
  const int cnt = gb - ga;
  const int e0 = ga + cnt * part / kp, e1 = ga + cnt * (part + 1) / kp;
  const int ne = e1 - e0;

  if (warp == 0) {
    tmem_alloc(smem_u32(&tmem_slot), SM_ROWS);
    tmem_relinquish();
  }
  if (tid == 0) {
    for (int i = 0; i < SM_STAGES; ++i) mbar_init(smem_u32(&mma_bar[i]), 1);
    abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (tid < SM_ROWS) {
    const int gr = rs * SM_ROWS + tid;
    const int panel = gr / P.bn == slot0 ? p0 : p1;
    bias_s[tid] = P.bias != nullptr && panel >= 0 ? __ldg(P.bias + panel * P.bn + gr % P.bn) : 0.f;
  }
  int *chunk = reinterpret_cast<int *>(sm + SM_CHUNK_OFF);
  const int32_t *entries = P.sched + sched_entries_offset_ints(P.n_groups);
  for (int i = tid; i < ne; i += SM_THREADS) {
    int c = __ldg(entries + e0 + i);
    if (c < 0 || c >= kc) {  // a corrupt list: flag it, read chunk 0
      atomicOr(&P.ctl->err, ERR_BAD_SCHED);
      c = 0;
    }
    chunk[i] = c;
  }

  // stage s <- entry i: this slice's 32 stream rows (they need only the entry's index), X rows
  // tt*128 .. +128 of the entry's chunk (zero beyond m and k)
  auto load_w = [&](int i, int s) {
    const uint32_t wsm = ring + s * SM_STAGE + SM_XB;
    const uint16_t *tile = P.wstream + ((int64_t)(e0 + i) * GROUP_FEATURES + rs * SM_ROWS) * CHUNK_COLS;
#pragma unroll
    for (int q = 0; q < SM_WB / 16 / SM_THREADS; ++q) {
      const int pc = tid + q * SM_THREADS, r = pc >> 3, j = pc & 7;
      cp_async16(wsm + sw_off(r, j), tile + r * CHUNK_COLS + j * 8, 16u);
    }
  };
  auto load_x = [&](int i, int s) {
    const int c = chunk[i];
    const uint32_t xs = ring + s * SM_STAGE;
#pragma unroll
    for (int q = 0; q < SM_XB / 16 / SM_THREADS; ++q) {
      const int pc = tid + q * SM_THREADS, r = pc >> 3, j = pc & 7;
      const int64_t t = (int64_t)tt * SM_TOK + r;
      const int col = c * CHUNK_COLS + j * 8;  // k is a multiple of 16: a piece is all in or all out
      const bool in = t < P.m && col < P.k;
      cp_async16(xs + sw_off(r, j), in ? P.X + t * P.ldx + col : P.X, in ? 16u : 0u);
    }
  };
  // the first stages' weight rows go out before the chunk indices are shared (they join the first
  // commit group, which only makes them complete no later than their stage needs them)
#pragma unroll
  for (int s = 0; s < SM_STAGES - 1; ++s)
    if (s < ne) load_w(s, s);
  tc_fence_before();
  __syncthreads();  // chunk indices, barriers and the TMEM address visible
  tc_fence_after();
  const uint32_t tmem = tmem_slot;
#pragma unroll
  for (int s = 0; s < SM_STAGES - 1; ++s) {
    if (s < ne) load_x(s, s);
    cp_async_commit();
  }

  bool ok = true;
  for (int i = 0; i < ne; ++i) {
    cp_async_wait<SM_STAGES - 2>();
    fence_proxy_async_smem();  // this thread's copies of entry i, visible to the tensor core
    __syncthreads();
    const int s = i % SM_STAGES;
    if (tid == 0) {
      tc_fence_after();
      const uint32_t xs = ring + s * SM_STAGE;
#pragma unroll
      for (int kk = 0; kk < CHUNK_COLS / 16; ++kk)
        umma_f16(tmem, smem_desc<128>(xs + kk * 32), smem_desc<128>(xs + SM_XB + kk * 32), SM_IDESC,
                 (i > 0 || kk > 0) ? 1u : 0u);
      tc_commit(smem_u32(&mma_bar[s]));
    }
    // refill the stage entry i - 1 used once its MMAs have read it
    const int nx = i + SM_STAGES - 1;
    if (nx < ne) {
      if (i >= 1 && !mbar_wait(smem_u32(&mma_bar[(i - 1) % SM_STAGES]), ((i - 1) / SM_STAGES) & 1u, &abort_flag,
                               P.timeout_ns))
        ok = false;
      load_w(nx, nx % SM_STAGES);
      load_x(nx, nx % SM_STAGES);
    }
    cp_async_commit();
  }
  cp_async_wait<0>();
  // every MMA done (they complete in order: the last commit covers them all)
  if (ne > 0 && !mbar_wait(smem_u32(&mma_bar[(ne - 1) % SM_STAGES]), ((ne - 1) / SM_STAGES) & 1u, &abort_flag,
                           P.timeout_ns))
    ok = false;
  if (!ok) atomicOr(&P.ctl->err, ERR_MMA_ACC);
  tc_fence_after();

  // warp w holds tokens 32 w .. 32 w + 31 (TMEM lanes), the slice's 32 group rows (columns)
  float v[SM_ROWS];
  if (ne > 0) {
    tmem_ld32(tmem + ((uint32_t)(32 * warp) << 16), v);
  } else {
#pragma unroll
    for (int c = 0; c < SM_ROWS; ++c) v[c] = 0.f;
  }
  const int r_own = 32 * warp + lane;
  if (kp == 1) {
    const int64_t t = (int64_t)tt * SM_TOK + r_own;
    if (t < P.m) {
#pragma unroll
      for (int run = 0; run < SM_ROWS / 8; ++run) {
        const int gr = rs * SM_ROWS + run * 8;  // the run's first group row; a run stays inside one panel
        const int panel = gr / P.bn == slot0 ? p0 : p1;
        if (panel >= 0) finish8<GELU, F32>(v + run * 8, bias_s + run * 8, panel * P.bn + gr % P.bn, t, P);
      }
    }
  } else {
    __syncthreads();  // every thread is past its last copy: the ring takes the partial tile
    float *pt = reinterpret_cast<float *>(sm);
#pragma unroll
    for (int c = 0; c < SM_ROWS; c += 4)
      *reinterpret_cast<float4 *>(pt + r_own * SM_PSTRIDE + c) = make_float4(v[c], v[c + 1], v[c + 2], v[c + 3]);
    cluster_sync();
    // rows part * 128 / kp ..: the kp partial tiles added in rank order, then the epilogue
    const int rows = SM_TOK / kp, r0 = part * rows;
    for (int it = tid; it < rows * (SM_ROWS / 8); it += SM_THREADS) {
      const int r = r0 + it / (SM_ROWS / 8), run = it % (SM_ROWS / 8);
      const int64_t t = (int64_t)tt * SM_TOK + r;
      const int gr = rs * SM_ROWS + run * 8;
      const int panel = gr / P.bn == slot0 ? p0 : p1;
      if (t >= P.m || panel < 0) continue;
      const uint32_t off = smem_u32(pt + r * SM_PSTRIDE + run * 8);
      // every part's values requested first (one remote latency), then added in rank order
      float4 lo[8], hi[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        if (q < kp) {
          const uint32_t rem = mapa_rank(off, (uint32_t)q);
          lo[q] = ld_cluster_f4(rem);
          hi[q] = ld_cluster_f4(rem + 16);
        }
      }
      float y[8] = {lo[0].x, lo[0].y, lo[0].z, lo[0].w, hi[0].x, hi[0].y, hi[0].z, hi[0].w};
#pragma unroll
      for (int q = 1; q < 8; ++q) {
        if (q < kp) {
          y[0] += lo[q].x; y[1] += lo[q].y; y[2] += lo[q].z; y[3] += lo[q].w;
          y[4] += hi[q].x; y[5] += hi[q].y; y[6] += hi[q].z; y[7] += hi[q].w;
        }
      }
      finish8<GELU, F32>(y, bias_s + run * 8, panel * P.bn + gr % P.bn, t, P);
    }
    cluster_sync();  // no CTA leaves while another still reads its partial tile
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, SM_ROWS);
}

}  // namespace

// ------------------------------------------------------------------------------------ host side

cudaError_t launch_linear(const CUtensorMap &tmX, const CUtensorMap &tmW, const LinearParams &P, int grid,
                          cudaStream_t s) {
  static bool attr_done[64] = {false};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64 && !attr_done[dev]) {
    for (auto k : {bsr_linear_kernel<false, false, false>, bsr_linear_kernel<true, false, false>,
                   bsr_linear_kernel<false, true, false>, bsr_linear_kernel<true, true, false>}) {
      cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, Smem<false>::BYTES);
      if (e != cudaSuccess) return e;
    }
    for (auto k : {bsr_linear_kernel<false, false, true>, bsr_linear_kernel<true, false, true>,
                   bsr_linear_kernel<false, true, true>, bsr_linear_kernel<true, true, true>}) {
      cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, Smem<true>::BYTES);
      if (e != cudaSuccess) return e;
    }
    attr_done[dev] = true;
  }
  // long K (at least DEEP_MIN_CHUNKS entries per unit): the seven-stage variant
  const bool deep = sched_chunks(P.k) >= DEEP_MIN_CHUNKS && P.S >= DEEP_MIN_CHUNKS;
  auto kern = deep ? (P.gelu ? (P.y_f32 ? bsr_linear_kernel<true, true, true> : bsr_linear_kernel<true, false, true>)
                             : (P.y_f32 ? bsr_linear_kernel<false, true, true> : bsr_linear_kernel<false, false, true>))
                   : (P.gelu ? (P.y_f32 ? bsr_linear_kernel<true, true, false> : bsr_linear_kernel<true, false, false>)
                             : (P.y_f32 ? bsr_linear_kernel<false, true, false> : bsr_linear_kernel<false, false, false>));
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(NUM_THREADS);
  cfg.dynamicSmemBytes = deep ? Smem<true>::BYTES : Smem<false>::BYTES;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e = cudaLaunchKernelEx(&cfg, kern, tmX, tmW, P);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

cudaError_t launch_linear_chain(const ChainParams &C, int grid, cudaStream_t s) {
  static bool attr_done[64] = {false};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64 && !attr_done[dev]) {
    cudaError_t e = cudaFuncSetAttribute(bsr_linear_chain_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         Smem<false>::BYTES);
    if (e != cudaSuccess) return e;
    attr_done[dev] = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(NUM_THREADS);
  cfg.dynamicSmemBytes = Smem<false>::BYTES;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e = cudaLaunchKernelEx(&cfg, bsr_linear_chain_kernel, C);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

cudaError_t launch_linear_small(LinearParams P, int num_sms, cudaStream_t s) {
  static bool attr_done[64] = {false};
  const int kc = sched_chunks(P.k);
  const size_t smem = (size_t)SM_CHUNK_OFF + (size_t)kc * sizeof(int) + 1024;  // + alignment slack
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64 && !attr_done[dev]) {
    // the largest request: kc <= 1024 chunk indices
    const int most = SM_CHUNK_OFF + 1024 * (int)sizeof(int) + 1024;
    for (auto k : {bsr_linear_small_kernel<false, false>, bsr_linear_small_kernel<true, false>,
                   bsr_linear_small_kernel<false, true>, bsr_linear_small_kernel<true, true>}) {
      cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, most);
      if (e != cudaSuccess) return e;
    }
    attr_done[dev] = true;
  }
  const int64_t ctas = ((P.m + SM_TOK - 1) / SM_TOK) * (int64_t)P.n_groups * SM_SLICES;
  // K parts: double while the grid stays resident at two CTAs per SM (the ring's shared memory)
  // and each part keeps at least 8 chunks. An entry costs a CTA ~0.45 us at batch 1 and the
  // cluster's reduction (two cluster barriers, remote reads) ~2.7 us, so shorter parts lose.
  int kp = 1;
  while (kp < 8 && ctas * kp * 2 <= 2 * (int64_t)num_sms && kc / (2 * kp) >= 8) kp *= 2;
  P.kp = kp;
  auto kern = P.gelu ? (P.y_f32 ? bsr_linear_small_kernel<true, true> : bsr_linear_small_kernel<true, false>)
                     : (P.y_f32 ? bsr_linear_small_kernel<false, true> : bsr_linear_small_kernel<false, false>);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(ctas * kp));
  cfg.blockDim = dim3(SM_THREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)kp;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = kp > 1 ? 1 : 0;  // no cluster when K is not cut
  cudaError_t e = cudaLaunchKernelEx(&cfg, kern, P);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

cudaError_t launch_split_reduce(const ReduceParams &R, int64_t threads, cudaStream_t s) {
  int64_t blocks = (threads + 255) / 256;
  if (blocks < 1) blocks = 1;
  if (blocks > 4096) blocks = 4096;
  split_reduce_kernel<<<(unsigned)blocks, 256, 0, s>>>(R);
  return cudaGetLastError();
}

}  // namespace lpvit
