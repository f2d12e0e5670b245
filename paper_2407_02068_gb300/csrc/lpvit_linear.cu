// Block-sparse linear Y = act(X W~^T + bias) on sm_103a (Sec. 3.1 block mask, Sec. 3.3
// block-sparse matmul: one block matmul per kept block and token tile, nothing for removed
// blocks). The kernel is compiled per block width BK (input columns of a block: 16, 32 or 64);
// the block height only decides which rows of a group tile the pack left zero.
//
// Work unit = 256 tokens x one 128-feature group of row panels (x one slice of the group's block
// columns when the problem is too small to fill the GPU); the work list's group table names the
// panels of each group and the epilogue maps a group row to its output feature through it.
// Per CTA (one per SM, persistent):
//   warp 0      producer: takes units from a global atomic queue, walks the unit's work-list
//               entries and, per entry (one block column j), loads the X tile [256 tokens x bk]
//               (TMA tensor copy) and the entry's 128 x bk group tile from the work list's weight
//               stream (one bulk copy), for a batch of entries at a time, one lane per copy.
//   warp 1      MMA issuer: per entry and per 16-wide k step, one tcgen05 MMA (M = 128, N = 256,
//               K = 16, both operands from shared memory): D[128 group rows x 256 tokens] +=
//               W_tile * X_tile^T, fp32 in TMEM. The W tile covers the whole group, with zero rows
//               for the slots whose panel keeps no block at this column.
//   warps 2..17 epilogue: TMEM -> registers, + bias, optional exact GELU, rounding to the output
//               type, stores of 64-byte row segments; split slices are summed in slice order
//               by the last slice to finish (ticket), which makes the result deterministic.
// Accumulators are double-buffered in TMEM (2 x 256 columns) so the epilogue of one unit overlaps
// the MMAs of the next. Every wait is bounded: on timeout the CTA records an error bit, drains its
// own copies and MMAs, frees TMEM and returns.
#include <cstdint>
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "lpvit_device.cuh"

namespace lpvit {

template <int BK>
struct Cfg {
  static constexpr int MP = GROUP_FEATURES;                 // MMA M: the group's 128 features
  static constexpr int KSTEPS = BK / 16;                    // 16-wide k steps per block column
  static constexpr int ROW_BYTES = BK * 2;                  // bytes of one tile row (bf16)
  static constexpr int TT = TOKENS_PER_TILE;                // MMA N: tokens per unit
  static constexpr int BUF_COLS = TT;                       // TMEM columns per accumulator buffer
  static constexpr int X_BYTES = TT * ROW_BYTES;            // X tile [256 x bk]
  static constexpr int A_BYTES = MP * ROW_BYTES;            // W tile [128 x bk]
  static constexpr int STAGE_BYTES = X_BYTES + A_BYTES;
  static constexpr int NSTAGES = 196608 / STAGE_BYTES;      // 192 KB of stages
  static constexpr int UR = 4;                              // unit-info ring depth
  // most entries per lane-parallel copy batch: the producer waits until that many stages are free,
  // so a batch trades its fixed issue cost against idle stages (measured best: 4 of 16, 3 of 8)
  static constexpr int BATCH = NSTAGES >= 16 ? 4 : (NSTAGES >= 8 ? 3 : 2);
  static constexpr int OPS = 2;                             // lane slots per entry: X tile, W tile
  static constexpr int NBMAX = BATCH < 32 / OPS ? BATCH : 32 / OPS;  // entries per batch
  static constexpr uint32_t IDESC = idesc_bf16(MP, TT);
  static_assert(A_BYTES == stream_tile_bytes(BK), "weight-stream tile geometry");
  static_assert(2 * BUF_COLS == 512, "two accumulator buffers fill the 512 TMEM columns");
  static_assert(NSTAGES >= 4, "pipeline depth");
  static_assert(X_BYTES % 1024 == 0 && A_BYTES % 1024 == 0, "tiles stay on their swizzle alignment");
};

constexpr int MMA_WARPS = 1;       // one MMA issuer
constexpr int FIRST_EPI = 1 + MMA_WARPS;
constexpr int EPI_WARPS = 16;      // four per TMEM lane quarter
static_assert(EPI_WARPS % 4 == 0, "epilogue warps come in whole sets of four lane quarters");
constexpr int NUM_THREADS = 32 * (FIRST_EPI + EPI_WARPS);   // 576
constexpr int MAX_GROUPS = 512;    // n <= 65536

struct UnitInfo {
  int tt, g, s, nsl, e0, e1, touched, pad;
};


template <int BK>
struct Smem {
  // stages first (1024-byte aligned), then the control area
  static constexpr int CTRL_OFF = Cfg<BK>::NSTAGES * Cfg<BK>::STAGE_BYTES;
  static constexpr int NS = Cfg<BK>::NSTAGES, UR = Cfg<BK>::UR;
  static constexpr int BAR_OFF = CTRL_OFF;
  // barriers: full[NS], empty[NS], accf[2], acce[2], unitf[UR], unite[UR], drain, episync
  static constexpr int NBARS = 2 * NS + 4 + 2 * UR + 2;
  static constexpr int RING_OFF = (BAR_OFF + 8 * NBARS + 31) / 32 * 32;
  static constexpr int SLICE_OFF = RING_OFF + (int)sizeof(UnitInfo) * UR;
  static constexpr int GENT_OFF = SLICE_OFF + 4 * (MAX_GROUPS + 1);  // the group entry table, staged
  static constexpr int MISC_OFF = GENT_OFF + 4 * (MAX_GROUPS + 1);
  static constexpr int EPI_OFF = (MISC_OFF + 64 + 127) / 128 * 128;
  static constexpr int EPI_TILE = 16 * 80;  // per epilogue warp: 16 token rows x 32 bf16, rows padded to 80 B
  static constexpr int END = EPI_OFF + EPI_WARPS * EPI_TILE;
  static constexpr int BYTES = END + 1024;  // + alignment slack for the dynamic smem base
  static_assert(BYTES <= 227 * 1024, "shared memory per CTA");
};

// Epilogue of one 32 x 32 block held by a warp: y[i] = accumulator of token tok_base + i for the
// lane's output feature fl (-1: a group row without a panel; turned into the output in place), bb =
// that feature's bias (0 without one). Lanes 8c .. 8c + 7 hold consecutive features of one row panel.
// Adds the bias, applies GELU, rounds, adds the bf16 residual if there is one (rounding again), and
// stores rows [tok_base, min(tok_base + 32, m)).
// bf16 output is staged through this warp's shared tile (rows padded to 80 bytes, conflict-free) so
// that every token row leaves as 16-byte vector stores; fp32 output is stored directly (a warp
// writes 128 contiguous bytes per token).
__device__ __forceinline__ void emit32(float (&y)[32], float bb, int fl, int64_t tok_base,
                                       const LinearParams &P, uint8_t *tile) {
  const int lane = threadIdx.x & 31;
  const int f = fl;
  const bool fvalid = fl >= 0;
  const int64_t left = P.m - tok_base;
  const int rows = left >= 32 ? 32 : (left > 0 ? (int)left : 0);
  if (P.gelu) {
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      // exact GELU, t * Phi(t); where 1 + erf cancels (t < -3) the error is a few ulps of 1 times t / 2
      const float t = y[i] + bb;
      y[i] = 0.5f * t * (1.f + erff(t * 0.70710678118654752440f));
    }
  } else {
#pragma unroll
    for (int i = 0; i < 32; ++i) y[i] += bb;
  }
  if (P.y_f32) {
    float *dst = static_cast<float *>(P.Y) + tok_base * P.ldy + f;
    if (fvalid) {
#pragma unroll
      for (int i = 0; i < 32; ++i)
        if (i < rows) dst[(int64_t)i * P.ldy] = y[i];
    }
    return;
  }
  __nv_bfloat16 *t = reinterpret_cast<__nv_bfloat16 *>(tile);
  const int ch = lane & 3;
  const int fch = __shfl_sync(0xffffffffu, fl, 8 * ch);  // first feature of the lane's 8-feature chunk
  const bool cvalid = fch >= 0;
#pragma unroll
  for (int half = 0; half < 2; ++half) {  // 16 token rows at a time through the warp's tile
#pragma unroll
    for (int i = 0; i < 16; ++i) t[i * 40 + lane] = __float2bfloat16_rn(y[16 * half + i]);
    __syncwarp();
#pragma unroll
    for (int it = 0; it < 2; ++it) {
      const int rt = 8 * it + (lane >> 2), row = 16 * half + rt;
      int4 val = *reinterpret_cast<const int4 *>(tile + rt * 80 + ch * 16);
      if (row < rows && cvalid) {
        if (P.R != nullptr) {
          // + the residual, each sum rounded to bf16 (a plain load: R may be Y itself, read and then
          // written by this thread only)
          const int4 rv = *reinterpret_cast<const int4 *>(P.R + (tok_base + row) * P.ldr + fch);
          __nv_bfloat16 *a = reinterpret_cast<__nv_bfloat16 *>(&val);
          const __nv_bfloat16 *b = reinterpret_cast<const __nv_bfloat16 *>(&rv);
#pragma unroll
          for (int e = 0; e < 8; ++e) a[e] = __float2bfloat16_rn(__bfloat162float(a[e]) + __bfloat162float(b[e]));
        }
        __nv_bfloat16 *dst = static_cast<__nv_bfloat16 *>(P.Y) + (tok_base + row) * P.ldy + fch;
        if (P.y_vec16) {
          *reinterpret_cast<int4 *>(dst) = val;
        } else {
          const __nv_bfloat16 *src = reinterpret_cast<const __nv_bfloat16 *>(&val);
#pragma unroll
          for (int e = 0; e < 8; ++e) dst[e] = src[e];
        }
      }
    }
    __syncwarp();
  }
}


// The MMAs of one work-list entry, issued by one elected thread: for every 16-wide k step,
// D[128 x 256] (+)= W_tile[128 x 16] * X_tile[256 x 16]^T, both tiles in the stage (X first).
template <int BK>
__device__ __forceinline__ void issue_entry(uint32_t st_u32, uint32_t dbase, uint32_t accumulate) {
  using C = Cfg<BK>;
#pragma unroll
  for (int kk = 0; kk < C::KSTEPS; ++kk) {
    const uint64_t bdesc = smem_desc<C::ROW_BYTES>(st_u32 + kk * 32);
    const uint64_t adesc = smem_desc<C::ROW_BYTES>(st_u32 + C::X_BYTES + kk * 32);
    umma_f16(dbase, adesc, bdesc, C::IDESC, (kk > 0 || accumulate) ? 1u : 0u);
  }
}

template <int BK>
__global__ void __launch_bounds__(NUM_THREADS, 1)
bsr_linear_kernel(const __grid_constant__ CUtensorMap tmX, const LinearParams P) {
  using C = Cfg<BK>;
  using L = Smem<BK>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t smem_base = smem_u32(smem);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  const uint32_t bar0 = smem_base + L::BAR_OFF;
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (L::NS + s); };
  auto accf_bar = [&](int b) { return bar0 + 8u * (2 * L::NS + b); };
  auto acce_bar = [&](int b) { return bar0 + 8u * (2 * L::NS + 2 + b); };
  auto unitf_bar = [&](int u) { return bar0 + 8u * (2 * L::NS + 4 + u); };
  auto unite_bar = [&](int u) { return bar0 + 8u * (2 * L::NS + 4 + L::UR + u); };
  const uint32_t drain_bar = bar0 + 8u * (2 * L::NS + 4 + 2 * L::UR);
  const uint32_t episync_bar = drain_bar + 8u;
  UnitInfo *ring = reinterpret_cast<UnitInfo *>(smem + L::RING_OFF);
  int *slice_ptr = reinterpret_cast<int *>(smem + L::SLICE_OFF);
  int *gent_s = reinterpret_cast<int *>(smem + L::GENT_OFF);
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + L::MISC_OFF);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(smem + L::MISC_OFF + 4);
  volatile int *last_flag = reinterpret_cast<volatile int *>(smem + L::MISC_OFF + 8);
  volatile int *never_flag = reinterpret_cast<volatile int *>(smem + L::MISC_OFF + 12);  // stays 0

  const int32_t *gent = P.sched + SCHED_HDR_INTS;
  const int32_t *entries = P.sched + sched_entries_offset_ints(P.n_groups);
  const int32_t *gpan = P.sched + sched_gpan_offset_ints(P.n_groups);
  const uint64_t tmo = P.timeout_ns;

  // ---------------------------------------------------------------- prologue
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), 512);
    tmem_relinquish();
  }
  if (tid == 0) {
    for (int s = 0; s < L::NS; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), MMA_WARPS);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(accf_bar(b), MMA_WARPS);
      mbar_init(acce_bar(b), EPI_WARPS);
    }
    for (int u = 0; u < L::UR; ++u) {
      mbar_init(unitf_bar(u), 1);
      mbar_init(unite_bar(u), EPI_WARPS);
    }
    mbar_init(drain_bar, MMA_WARPS);
    mbar_init(episync_bar, EPI_WARPS);
    *abort_flag = 0;
    *last_flag = 0;
    *never_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0 && lane == 0) prefetch_tensormap(&tmX);
  // the work list must be this weight's plan: group count, shape and block width
  const bool sched_ok = P.sched[3] == 0 && P.sched[1] == P.n_groups && P.sched[4] == P.n && P.sched[5] == P.k &&
                        P.sched[6] == P.bn && P.sched[7] == BK;
  if (warp == 2) {
    // slices per group = max(1, ceil(entries / S)); exclusive prefix into slice_ptr
    int run = 0;
    for (int base = 0; base < P.n_groups; base += 32) {
      const int g = base + lane;
      int c = 0;
      if (g < P.n_groups) {
        const int cnt = gent[g + 1] - gent[g];
        c = cnt <= 0 ? 1 : (cnt + P.S - 1) / P.S;
      }
      int incl = c;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int t = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += t;
      }
      if (g < P.n_groups) slice_ptr[g] = run + incl - c;
      run += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (lane == 0) slice_ptr[P.n_groups] = run;
    for (int g = lane; g <= P.n_groups; g += 32) gent_s[g] = gent[g];
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int total_slices = slice_ptr[P.n_groups];
  const uint32_t total_units = sched_ok ? (uint32_t)P.n_tt * (uint32_t)total_slices : 0u;
  if (!sched_ok && tid == 0) atomicOr(&P.ctl->err, P.sched[3] ? ERR_SCHED_OVERFLOW : ERR_BAD_SCHED);

  if (warp == 0) {
    // ============================================================== producer
    // Unit i is decoded (shared-memory tables) and its first 32 entry records are loaded while unit
    // i - 1 is issued, and the queue index of unit i + 1 is fetched then; within a unit the next 32
    // records are loaded while the current ones are issued. No global round trip sits on the path.
    uint32_t it = 0, ui = 0;
    bool ok = true;
    struct Unit {
      int tt, g, s, nsl, e0, e1;
    };
    auto decode = [&](uint32_t u) {  // shared-memory tables only
      Unit d;
      d.tt = (int)(u / (uint32_t)total_slices);
      const int rr = (int)(u % (uint32_t)total_slices);
      int lo = 0, hi = P.n_groups - 1;  // group g with slice_ptr[g] <= rr < slice_ptr[g+1]
      while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (slice_ptr[mid] <= rr) lo = mid;
        else hi = mid - 1;
      }
      d.g = lo;
      d.s = rr - slice_ptr[lo];
      d.nsl = slice_ptr[lo + 1] - slice_ptr[lo];
      const int ge0 = gent_s[lo], ge1 = gent_s[lo + 1];
      d.e0 = min(ge0 + d.s * P.S, ge1);
      d.e1 = min(d.e0 + P.S, ge1);
      return d;
    };
    auto first_records = [&](const Unit &d, int &w, int &t) {
      w = 0;
      t = -1;
      if (d.e0 + lane < d.e1) {
        const int32_t *ep = entries + (int64_t)(d.e0 + lane) * ENTRY_INTS;
        w = ep[0];
        t = ep[ENTRY_TILE_WORD];
      }
    };
    uint32_t fetched = 0;
    if (lane == 0) fetched = atomicAdd(&P.ctl->next_unit, 1u);
    uint32_t u_cur = __shfl_sync(0xffffffffu, fetched, 0);
    Unit cur = {0, 0, 0, 1, 0, 0};
    int w0c = 0, toffc = -1;
    if (u_cur < total_units) {
      cur = decode(u_cur);
      first_records(cur, w0c, toffc);
      if (lane == 0) fetched = atomicAdd(&P.ctl->next_unit, 1u);
    }
    while (true) {
      const uint32_t u = u_cur;
      const uint32_t slot = ui % L::UR, uph = (ui / L::UR) & 1u;
      if (!mbar_wait(unite_bar(slot), uph ^ 1u, abort_flag, tmo)) {
        ok = false;
        if (lane == 0) atomicOr(&P.ctl->err, ERR_PRODUCER_UNIT);
        break;
      }
      if (u >= total_units) {
        if (lane == 0) {
          ring[slot].tt = -1;
          mbar_arrive(unitf_bar(slot));
        }
        break;
      }
      const int tt = cur.tt, e0 = cur.e0, e1 = cur.e1;
      // every entry keeps a block of the group, so the accumulator is written iff there is one
      const unsigned tmask = e1 > e0 ? 1u : 0u;
      if (lane == 0) {
        UnitInfo inf;
        inf.tt = tt; inf.g = cur.g; inf.s = cur.s; inf.nsl = cur.nsl; inf.e0 = e0; inf.e1 = e1;
        inf.touched = (int)tmask;
        inf.pad = 0;
        ring[slot] = inf;
        mbar_arrive(unitf_bar(slot));
      }
      // the next unit: decode it, start loading its first records, fetch the one after
      const uint32_t u_nx = __shfl_sync(0xffffffffu, fetched, 0);
      Unit nxt = {0, 0, 0, 1, 0, 0};
      int w0x = 0, toffx = -1;
      if (u_nx < total_units) {
        nxt = decode(u_nx);
        first_records(nxt, w0x, toffx);
        if (lane == 0) fetched = atomicAdd(&P.ctl->next_unit, 1u);
      }
      int w0n = w0c, toffn = toffc;  // records of entries base + lane, loaded one chunk ahead
      for (int base = e0; base < e1 && ok; base += 32) {
        const int w0 = w0n, toff = toffn;
        w0n = 0;
        toffn = -1;
        if (base + 32 + lane < e1) {
          const int32_t *ep = entries + (int64_t)(base + 32 + lane) * ENTRY_INTS;
          w0n = ep[0];
          toffn = ep[ENTRY_TILE_WORD];
        }
        const int cnt = min(32, e1 - base);
        for (int i = 0; i < cnt && ok;) {
          // One batch = NBMAX consecutive entries. Lanes 2k and 2k+1 issue the two copies of entry k
          // (its X tile, its weight tiles), all in one instruction: a thread's bulk copies are
          // processed one after another, copies from different threads overlap.
          const int nb = min(C::NBMAX, cnt - i);
          bool wok = true;
          if (lane < nb) {
            const uint32_t itk = it + lane;
            wok = mbar_wait(empty_bar(itk % L::NS), ((itk / L::NS) & 1u) ^ 1u, abort_flag, tmo);
          }
          if (!__all_sync(0xffffffffu, wok)) {
            ok = false;
            if (lane == 0) atomicOr(&P.ctl->err, ERR_PRODUCER_EMPTY);
            break;
          }
          const int k2 = lane >> 1;
          const int src = min(i + k2, 31);
          const int wk = __shfl_sync(0xffffffffu, w0, src);
          const int tk = __shfl_sync(0xffffffffu, toff, src);
          uint32_t mm = ((uint32_t)wk >> 16) != 0u ? 1u : 0u;  // the entry keeps a block of the group
          // a tile range outside the stream region means a corrupt work list: flag it, load no weights
          const bool tiles_ok = tk >= 0 && (int64_t)tk + __popc(mm) <= P.stream_tiles;
          if (!tiles_ok) mm = 0;
          const uint32_t stk = (it + k2) % L::NS;
          const uint32_t st_u32 = smem_base + stk * C::STAGE_BYTES;
          if (k2 < nb && (lane & 1) == 0) {
            if (!tiles_ok) atomicOr(&P.ctl->err, ERR_BAD_SCHED);
            mbar_arrive_expect_tx(full_bar(stk), C::X_BYTES + __popc(mm) * C::A_BYTES);
          }
          __syncwarp();
          if (k2 < nb) {
            if ((lane & 1) == 0)
              tma_load_2d(st_u32, &tmX, (wk & 0xffff) * BK, tt * C::TT, full_bar(stk));
            else if (mm)
              bulk_load(st_u32 + C::X_BYTES, P.wstream + (int64_t)tk * C::A_BYTES, __popc(mm) * C::A_BYTES,
                        full_bar(stk));
          }
          __syncwarp();
          it += nb;
          i += nb;
        }
      }
      if (!ok) break;
      ++ui;
      u_cur = u_nx;
      cur = nxt;
      w0c = w0x;
      toffc = toffx;
    }
    if (!ok && lane == 0) *abort_flag = 1;
    // queue bookkeeping: the last CTA to leave resets the counters for the next launch
    if (lane == 0) {
      __threadfence();
      if (atomicAdd(&P.ctl->done_ctas, 1u) == gridDim.x - 1) {
        P.ctl->next_unit = 0;
        P.ctl->done_ctas = 0;
        __threadfence();
      }
    }
    // make sure no TMA write into this CTA's smem is still in flight
    const uint32_t first = it > (uint32_t)L::NS ? it - L::NS : 0u;
    for (uint32_t i = first; i < it; ++i)
      if (!mbar_wait(full_bar(i % L::NS), (i / L::NS) & 1u, never_flag, tmo)) break;
  } else if (warp < FIRST_EPI) {
    // ============================================================== MMA issuer
    // Arrives on a stage's empty barrier once per entry: a commit when it issued MMAs there.
    uint32_t it = 0, ui = 0;
    bool ok = true;
    while (ok) {
      const uint32_t slot = ui % L::UR, uph = (ui / L::UR) & 1u;
      if (!mbar_wait(unitf_bar(slot), uph, abort_flag, tmo)) {
        ok = false;
        if (lane == 0) atomicOr(&P.ctl->err, ERR_MMA_UNIT);
        break;
      }
      const UnitInfo inf = ring[slot];
      if (inf.tt < 0) break;
      const uint32_t buf = ui & 1u, aph = (ui >> 1) & 1u;
      if (!mbar_wait(acce_bar(buf), aph ^ 1u, abort_flag, tmo)) {
        ok = false;
        if (lane == 0) atomicOr(&P.ctl->err, ERR_MMA_ACC);
        break;
      }
      tc_fence_after();
      const uint32_t dbase = tmem_base + buf * C::BUF_COLS;
      uint32_t touched = 0;
      for (int e = inf.e0; e < inf.e1; ++e) {
        const uint32_t stage = it % L::NS, ph = (it / L::NS) & 1u;
        if (!mbar_wait(full_bar(stage), ph, abort_flag, tmo)) {
          ok = false;
          if (lane == 0) atomicOr(&P.ctl->err, ERR_MMA_FULL);
          break;
        }
        tc_fence_after();
        // every entry keeps a block of its group, so every stage holds a W tile (a work list whose
        // tile range is corrupt has its error bit set and its stage's weights left stale)
        const uint32_t st_u32 = smem_base + stage * C::STAGE_BYTES;
        if (elect_one()) {
          issue_entry<BK>(st_u32, dbase, touched);
          tc_commit(empty_bar(stage));
        }
        __syncwarp();
        touched = 1;
        ++it;
      }
      if (!ok) break;
      if (elect_one()) {
        if (touched) tc_commit(accf_bar(buf));
        else mbar_arrive(accf_bar(buf));
      }
      __syncwarp();
      ++ui;
    }
    if (!ok && lane == 0) *abort_flag = 1;
    // wait for every MMA this thread issued before TMEM can be freed
    if (elect_one()) tc_commit(drain_bar);
    __syncwarp();
    if (!mbar_wait(drain_bar, 0, never_flag, tmo) && lane == 0) atomicOr(&P.ctl->err, ERR_DRAIN);
  } else {
    // ============================================================== epilogue
    // A unit's accumulator is 128 features (TMEM lanes) x 256 tokens (columns). Per TMEM lane
    // quarter (32 features) it forms 8 blocks of 32 tokens; the quarter's EPI_WARPS / 4 warps take
    // them in turn.
    const int ew = warp - FIRST_EPI;             // 0 .. EPI_WARPS - 1
    const int q = warp & 3;                      // TMEM lane quarter this warp may access
    const int wq = ew >> 2;                      // this warp's turn within its quarter
    constexpr int QBLK = C::TT / 32;             // blocks per lane quarter
    uint32_t ui = 0, sync_phase = 0;
    uint8_t *epi_tile = smem + L::EPI_OFF + ew * L::EPI_TILE;
    while (true) {
      const uint32_t slot = ui % L::UR, uph = (ui / L::UR) & 1u;
      if (!mbar_wait(unitf_bar(slot), uph, abort_flag, tmo)) {
        if (lane == 0) { atomicOr(&P.ctl->err, ERR_EPI_UNIT); *abort_flag = 1; }
        break;
      }
      const UnitInfo inf = ring[slot];
      if (inf.tt < 0) break;
      // this lane's group row 32 q + lane is row (32 q + lane) % bn of the panel in slot (32 q + lane) / bn;
      // its feature and bias are loaded while the accumulator is still being computed
      const int grow = 32 * q + lane;
      const int panel = __ldg(gpan + (int64_t)inf.g * MAX_GROUP_PANELS + grow / P.bn);
      const int fl = panel >= 0 ? panel * P.bn + grow % P.bn : -1;
      const float bb = (P.bias != nullptr && fl >= 0) ? __ldg(P.bias + fl) : 0.f;
      const uint32_t buf = ui & 1u, aph = (ui >> 1) & 1u;
      if (!mbar_wait(accf_bar(buf), aph, abort_flag, tmo)) {
        if (lane == 0) { atomicOr(&P.ctl->err, ERR_EPI_ACC); *abort_flag = 1; }
        break;
      }
      tc_fence_after();
      const bool split = inf.nsl > 1;
      float *part = nullptr;
      if (split)
        part = P.partials + ((int64_t)inf.tt * total_slices + slice_ptr[inf.g] + inf.s) * (int64_t)(C::TT * 128);
#pragma unroll 1
      for (int j = wq; j < QBLK; j += EPI_WARPS / 4) {
        const int tok0 = 32 * j;  // first token of the block (its accumulator column)
        const uint32_t taddr = tmem_base + ((uint32_t)(32 * q) << 16) + buf * C::BUF_COLS + tok0;
        float v[32];
        if (inf.touched) {
          tmem_ld32(taddr, v);
        } else {
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] = 0.f;
        }
        if (split) {
          float4 *dst = reinterpret_cast<float4 *>(part + (int64_t)(32 * q + lane) * C::TT + tok0);
#pragma unroll
          for (int i = 0; i < 8; ++i) dst[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
        } else {
          emit32(v, bb, fl, (int64_t)inf.tt * C::TT + tok0, P, epi_tile);
        }
      }
      // accumulator buffer and unit slot are free again
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(acce_bar(buf));
        mbar_arrive(unite_bar(slot));
      }
      if (split) {
        // make the partial visible, take a ticket; the last slice sums all partials in order
        __threadfence();
        __syncwarp();
        if (lane == 0) mbar_arrive(episync_bar);
        if (!mbar_wait(episync_bar, sync_phase, abort_flag, tmo)) {
          if (lane == 0) { atomicOr(&P.ctl->err, ERR_EPI_UNIT); *abort_flag = 1; }
          break;
        }
        sync_phase ^= 1u;
        if (ew == 0 && lane == 0) {
          int32_t *tk = P.tickets + (int64_t)inf.tt * P.n_groups + inf.g;
          const int old = atomicAdd(tk, 1);
          const int last = old == inf.nsl - 1;
          if (last) atomicExch(tk, 0);
          *last_flag = last;
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(episync_bar);
        if (!mbar_wait(episync_bar, sync_phase, abort_flag, tmo)) {
          if (lane == 0) { atomicOr(&P.ctl->err, ERR_EPI_UNIT); *abort_flag = 1; }
          break;
        }
        sync_phase ^= 1u;
        const int last = *last_flag;
        if (last) {
          __threadfence();
          const float *base0 =
              P.partials + ((int64_t)inf.tt * total_slices + slice_ptr[inf.g]) * (int64_t)(C::TT * 128);
#pragma unroll 1
          for (int j = wq; j < QBLK; j += EPI_WARPS / 4) {
            const int tok0 = 32 * j;
            float v[32];
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] = 0.f;
            for (int s2 = 0; s2 < inf.nsl; ++s2) {
              const float4 *src = reinterpret_cast<const float4 *>(
                  base0 + (int64_t)s2 * (C::TT * 128) + (int64_t)(32 * q + lane) * C::TT + tok0);
#pragma unroll
              for (int i = 0; i < 8; ++i) {
                const float4 t = __ldcg(src + i);
                v[4 * i] += t.x; v[4 * i + 1] += t.y; v[4 * i + 2] += t.z; v[4 * i + 3] += t.w;
              }
            }
            emit32(v, bb, fl, (int64_t)inf.tt * C::TT + tok0, P, epi_tile);
          }
        }
      }
      ++ui;
    }
  }

  // ---------------------------------------------------------------- teardown
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem_base, 512);
}

// ------------------------------------------------------------------------------------ host side

template <int BK>
int smem_bytes() { return Smem<BK>::BYTES; }

template <int BK>
cudaError_t launch_linear_t(const CUtensorMap &tmX, const LinearParams &P, int grid, cudaStream_t s) {
  static bool attr_done[64] = {false};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64 && !attr_done[dev]) {
    cudaError_t e = cudaFuncSetAttribute(bsr_linear_kernel<BK>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         Smem<BK>::BYTES);
    if (e != cudaSuccess) return e;
    attr_done[dev] = true;
  }
  bsr_linear_kernel<BK><<<grid, NUM_THREADS, Smem<BK>::BYTES, s>>>(tmX, P);
  return cudaGetLastError();
}

cudaError_t launch_linear(int bk, const CUtensorMap &tmX, const LinearParams &P, int grid, cudaStream_t s) {
  switch (bk) {
    case 16: return launch_linear_t<16>(tmX, P, grid, s);
    case 32: return launch_linear_t<32>(tmX, P, grid, s);
    case 64: return launch_linear_t<64>(tmX, P, grid, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace lpvit
