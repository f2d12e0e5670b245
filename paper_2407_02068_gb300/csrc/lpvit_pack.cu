// Mask -> BSR pack and work-list build (Sec. 3.1 block mask; Sec. 1 / Sec. 3.3: only the kept
// blocks are stored, moved and multiplied).
//
// Blocks are bn output rows by bk input columns (Sec. 3.1 block mask; B_k x B_n in the notation of
// Sec. 3.3, whose weight is [N inputs x K outputs]).
// plan kernel (one CTA): per row panel r (bn rows), cnt[r] = number of kept blocks (warp
//   reductions); row_ptr = exclusive prefix sum of cnt (warp-shuffle scan + a scan of warp
//   totals); col_idx = kept block columns of each panel in ascending order (ballot compaction);
//   work list: the GEMM covers the weight in tiles of 256 output features by 64 input columns (a
//   "chunk"); panels are grouped 256 features (256 / bn panels) at a time, greedily by overlap of
//   the chunks in which they keep blocks (one warp; consecutive panels when that is not better);
//   for every group, one entry per chunk where any panel of the group keeps a block.
// copy kernel (grid-stride): blocks[t] = W[r*bn:(r+1)*bn, j*bk:(j+1)*bk], 16-byte vector copies,
//   bits unchanged; then the weight stream, entry by entry: the group's 256 rows over the chunk's
//   64 columns, row-major, removed blocks and empty slots zero.
#include <cstdint>
#include <cuda_runtime.h>

#include "lpvit_device.cuh"

namespace lpvit {

constexpr int PLAN_THREADS = 1024;
constexpr int PLAN_WARPS = PLAN_THREADS / 32;

// Exclusive block-wide scan of v[0..count) in shared memory (in place); returns the total.
// All threads of the CTA must call it.
__device__ int block_exclusive_scan(int *v, int count, int *warp_tot) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int per = (count + PLAN_THREADS - 1) / PLAN_THREADS;
  const int beg = min(count, tid * per), end = min(count, beg + per);
  int local = 0;
  for (int i = beg; i < end; ++i) local += v[i];
  int incl = local;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int t = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += t;
  }
  if (lane == 31) warp_tot[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    int w = warp_tot[lane];
    int wi = w;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int t = __shfl_up_sync(0xffffffffu, wi, o);
      if (lane >= o) wi += t;
    }
    warp_tot[lane] = wi - w;  // exclusive prefix of warp totals
    if (lane == 31) warp_tot[32] = wi;
  }
  __syncthreads();
  int run = warp_tot[warp] + incl - local;
  for (int i = beg; i < end; ++i) {
    const int c = v[i];
    v[i] = run;
    run += c;
  }
  const int total = warp_tot[32];
  __syncthreads();
  return total;
}

// Panel grouping runs when its bitmaps fit the plan's shared memory: at most GROUPING_MAX_PANELS
// row panels and GROUPING_MAX_WORDS words of per-panel column bitmaps.
constexpr int GROUPING_MAX_PANELS = 1024;
constexpr int GROUPING_MAX_WORDS = 8192;
__host__ __device__ inline bool grouping_on(int np, int kc, int gb) {
  const int W = (kc + 31) / 32;
  return gb >= 2 && np <= GROUPING_MAX_PANELS && (int64_t)np * W <= GROUPING_MAX_WORDS;
}

__device__ __forceinline__ int warp_sum(int v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Group the row panels, one warp. A group starts with the unassigned panel keeping the most blocks
// and then takes, gb - 1 times, the unassigned panel that adds the fewest chunks to the group's
// union (ties to the lower panel index). The work list has one entry per chunk of the union, so
// overlapping panels make fewer entries. The grouping is kept only if it gives fewer
// entries than consecutive panels; gpan is written either way.
__device__ void group_panels(const unsigned *__restrict__ bits, int W, const int *__restrict__ kcnt, int np,
                             int gb, int ng, unsigned *U, int *asg, int32_t *__restrict__ gpan) {
  const int lane = threadIdx.x & 31;
  for (int p = lane; p < np; p += 32) asg[p] = 0;
  int id_e = 0;  // entries of consecutive groups
  for (int g = lane; g < ng; g += 32)
    for (int w = 0; w < W; ++w) {
      unsigned u = 0;
      for (int p = 0; p < gb; ++p)
        if (g * gb + p < np) u |= bits[(g * gb + p) * W + w];
      id_e += __popc(u);
    }
  id_e = warp_sum(id_e);
  __syncwarp();
  int gr_e = 0;
  for (int g = 0; g < ng; ++g) {
    for (int sl = 0; sl < gb; ++sl) {
      int best = 0x7fffffff, bi = 0x7fffffff;
      for (int p = lane; p < np; p += 32) {
        if (asg[p]) continue;
        int sc = 0;
        if (sl == 0) {
          sc = -kcnt[p];
        } else {
          for (int w = 0; w < W; ++w) sc += __popc(bits[p * W + w] & ~U[w]);
        }
        if (sc < best || (sc == best && p < bi)) {
          best = sc;
          bi = p;
        }
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const int ob = __shfl_xor_sync(0xffffffffu, best, o), oi = __shfl_xor_sync(0xffffffffu, bi, o);
        if (ob < best || (ob == best && oi < bi)) {
          best = ob;
          bi = oi;
        }
      }
      const int pick = bi == 0x7fffffff ? -1 : bi;
      if (lane == 0) {
        gpan[g * MAX_GROUP_PANELS + sl] = pick;
        if (pick >= 0) asg[pick] = 1;
      }
      for (int w = lane; w < W; w += 32) {
        const unsigned add = pick >= 0 ? bits[pick * W + w] : 0u;
        U[w] = (sl == 0 ? 0u : U[w]) | add;
      }
      __syncwarp();
    }
    if (lane >= gb && lane < MAX_GROUP_PANELS) gpan[g * MAX_GROUP_PANELS + lane] = -1;
    int c = 0;
    for (int w = lane; w < W; w += 32) c += __popc(U[w]);
    gr_e += warp_sum(c);
    __syncwarp();
  }
  if (gr_e >= id_e) {
    for (int i = lane; i < ng * MAX_GROUP_PANELS; i += 32) {
      const int g = i / MAX_GROUP_PANELS, sl = i - g * MAX_GROUP_PANELS, r = g * gb + sl;
      gpan[i] = (sl < gb && r < np) ? r : -1;
    }
  }
}

// group_panels for up to 32 * FAST_NPL panels and FAST_W bitmap words, with the same rule and
// result: each lane keeps its candidates' bitmaps and kept counts in registers and every lane the
// group's union, so a step is register arithmetic, the warp argmin and FAST_W shuffles.
constexpr int FAST_NPL = 4, FAST_W = 4;
__device__ void group_panels_fast(const unsigned *__restrict__ bits, int W, const int *__restrict__ kcnt, int np,
                                  int gb, int ng, int32_t *__restrict__ gpan) {
  const int lane = threadIdx.x & 31;
  unsigned cb[FAST_NPL][FAST_W];
  int kc[FAST_NPL];
  unsigned alive = 0;  // bit i: candidate lane + 32 i is unassigned
#pragma unroll
  for (int i = 0; i < FAST_NPL; ++i) {
    const int p = lane + 32 * i;
    kc[i] = p < np ? kcnt[p] : 0;
    if (p < np) alive |= 1u << i;
#pragma unroll
    for (int w = 0; w < FAST_W; ++w) cb[i][w] = (p < np && w < W) ? bits[p * W + w] : 0u;
  }
  int id_e = 0;  // entries of consecutive groups
  for (int g = lane; g < ng; g += 32)
    for (int w = 0; w < W; ++w) {
      unsigned u = 0;
      for (int p = 0; p < gb; ++p)
        if (g * gb + p < np) u |= bits[(g * gb + p) * W + w];
      id_e += __popc(u);
    }
  id_e = warp_sum(id_e);
  int gr_e = 0;
  unsigned U[FAST_W];
  for (int g = 0; g < ng; ++g) {
#pragma unroll
    for (int w = 0; w < FAST_W; ++w) U[w] = 0u;
    for (int sl = 0; sl < gb; ++sl) {
      int best = 0x7fffffff, bi = 0x7fffffff;
#pragma unroll
      for (int i = 0; i < FAST_NPL; ++i) {
        if ((alive >> i) & 1u) {
          int sc = 0;
          if (sl == 0) {
            sc = -kc[i];
          } else {
#pragma unroll
            for (int w = 0; w < FAST_W; ++w) sc += __popc(cb[i][w] & ~U[w]);
          }
          if (sc < best) {  // candidates of a lane come in ascending index order
            best = sc;
            bi = lane + 32 * i;
          }
        }
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const int ob = __shfl_xor_sync(0xffffffffu, best, o), oi = __shfl_xor_sync(0xffffffffu, bi, o);
        if (ob < best || (ob == best && oi < bi)) {
          best = ob;
          bi = oi;
        }
      }
      const int pick = bi == 0x7fffffff ? -1 : bi;
      if (lane == 0) gpan[g * MAX_GROUP_PANELS + sl] = pick;
      if (pick >= 0) {
        const int owner = pick & 31, ip = pick >> 5;
        if (lane == owner) alive &= ~(1u << ip);
#pragma unroll
        for (int w = 0; w < FAST_W; ++w) {
          unsigned mine = 0;
#pragma unroll
          for (int i = 0; i < FAST_NPL; ++i)
            if (i == ip) mine = cb[i][w];
          U[w] |= __shfl_sync(0xffffffffu, mine, owner);
        }
      }
    }
    if (lane >= gb && lane < MAX_GROUP_PANELS) gpan[g * MAX_GROUP_PANELS + lane] = -1;
#pragma unroll
    for (int w = 0; w < FAST_W; ++w) gr_e += __popc(U[w]);  // the same in every lane
  }
  __syncwarp();
  if (gr_e >= id_e) {
    for (int i = lane; i < ng * MAX_GROUP_PANELS; i += 32) {
      const int g = i / MAX_GROUP_PANELS, sl = i - g * MAX_GROUP_PANELS, r = g * gb + sl;
      gpan[i] = (sl < gb && r < np) ? r : -1;
    }
  }
}

// Does panel r keep a block in chunk c (input columns [64 c, 64 c + 64))?
__device__ __forceinline__ bool chunk_kept(const uint8_t *__restrict__ mask, int r, int c, int kb, int bpc) {
  bool any = false;
  for (int q = 0; q < bpc; ++q) {
    const int j = c * bpc + q;
    any |= j < kb && mask[(int64_t)r * kb + j] != 0;
  }
  return any;
}

// The plan of one weight, computed by one CTA of PLAN_THREADS threads (plan_smem: plan_smem_bytes).
__device__ __forceinline__ void plan_body(const uint8_t *__restrict__ mask, int n, int k, int bn, int bk,
                                          int32_t *__restrict__ row_ptr, int32_t *__restrict__ col_idx, int cap,
                                          int32_t *__restrict__ sched, int *plan_smem) {
  const int np = n / bn, kb = k / bk;
  const int kc = sched_chunks(k);          // chunks of CHUNK_COLS input columns
  const int bpc = CHUNK_COLS / bk;         // blocks per chunk (bk divides CHUNK_COLS)
  const int gb = GROUP_FEATURES / bn;      // row panels per group
  const int ng = (n + GROUP_FEATURES - 1) / GROUP_FEATURES;
  const int W = (kc + 31) / 32;            // words of a panel's chunk bitmap
  const bool grouping = grouping_on(np, kc, gb);
  int *cnt = plan_smem;            // [np + 1]
  int *gcnt = cnt + np + 1;        // [ng + 1]
  int *warp_tot = gcnt + ng + 1;   // [33]
  int *kcnt = warp_tot + 33;       // [np] kept blocks per panel
  unsigned *bits = reinterpret_cast<unsigned *>(kcnt + np);  // grouping: [np][W] chunk bitmaps
  unsigned *U = bits + (grouping ? np * W : 0);              // grouping: [W] union of a group
  int *asg = reinterpret_cast<int *>(U + (grouping ? W : 0));  // grouping: [np] assigned flags
  int32_t *gpan = sched + sched_gpan_offset_ints(ng);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const unsigned lt = (1u << lane) - 1u;

  // 1. kept blocks per panel; chunk bitmaps for the grouping
  for (int r = warp; r < np; r += PLAN_WARPS) {
    int c = 0;
    for (int j = lane; j < kb; j += 32) c += mask[(int64_t)r * kb + j] != 0;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
    if (lane == 0) {
      cnt[r] = c;
      kcnt[r] = c;
    }
    if (grouping)
      for (int base = 0; base < kc; base += 32) {
        const int ch = base + lane;
        const unsigned bal = __ballot_sync(0xffffffffu, ch < kc && chunk_kept(mask, r, ch, kb, bpc));
        if (lane == 0) bits[r * W + base / 32] = bal;
      }
  }
  __syncthreads();
  // 2. row_ptr = exclusive scan
  const int nnzb = block_exclusive_scan(cnt, np, warp_tot);
  for (int r = tid; r < np; r += PLAN_THREADS) row_ptr[r] = cnt[r];
  if (tid == 0) {
    row_ptr[np] = nnzb;
    cnt[np] = nnzb;
  }
  __syncthreads();
  // 3. col_idx, ascending within each panel
  for (int r = warp; r < np; r += PLAN_WARPS) {
    int run = cnt[r];
    for (int base = 0; base < kb; base += 32) {
      const int j = base + lane;
      const bool keep = j < kb && mask[(int64_t)r * kb + j] != 0;
      const unsigned bal = __ballot_sync(0xffffffffu, keep);
      if (keep) {
        const int pos = run + __popc(bal & lt);
        if (pos < cap) col_idx[pos] = j;
      }
      run += __popc(bal);
    }
  }
  // 3b. group table: overlapping panels (one warp), or consecutive panels
  if (grouping) {
    if (warp == 0) {
      if (np <= 32 * FAST_NPL && W <= FAST_W) group_panels_fast(bits, W, kcnt, np, gb, ng, gpan);
      else group_panels(bits, W, kcnt, np, gb, ng, U, asg, gpan);
    }
  } else {
    for (int i = tid; i < ng * MAX_GROUP_PANELS; i += PLAN_THREADS) {
      const int g = i / MAX_GROUP_PANELS, sl = i - g * MAX_GROUP_PANELS, r = g * gb + sl;
      gpan[i] = (sl < gb && r < np) ? r : -1;
    }
  }
  __syncthreads();
  // 4a. entries per group: chunks where any panel of the group keeps a block
  for (int g = warp; g < ng; g += PLAN_WARPS) {
    int c = 0;
    for (int base = 0; base < kc; base += 32) {
      const int ch = base + lane;
      bool any = false;
      for (int p = 0; p < gb && ch < kc; ++p) {
        const int r = gpan[g * MAX_GROUP_PANELS + p];
        if (r >= 0) any |= chunk_kept(mask, r, ch, kb, bpc);
      }
      c += __popc(__ballot_sync(0xffffffffu, any));
    }
    if (lane == 0) gcnt[g] = c;
  }
  __syncthreads();
  const int total_entries = block_exclusive_scan(gcnt, ng, warp_tot);
  int32_t *gent = sched + SCHED_HDR_INTS;
  int32_t *entries = sched + sched_entries_offset_ints(ng);
  for (int g = tid; g < ng; g += PLAN_THREADS) gent[g] = gcnt[g];
  if (tid == 0) {
    gent[ng] = total_entries;
    sched[0] = nnzb;
    sched[1] = ng;
    sched[2] = total_entries;
    sched[3] = nnzb > cap ? 1 : 0;
    sched[4] = n;
    sched[5] = k;
    sched[6] = bn;
    sched[7] = bk;
    sched[8] = SCHED_VERSION;
    for (int i = 9; i < SCHED_HDR_INTS; ++i) sched[i] = 0;
  }
  // 4b. entries: the chunk index, in ascending order within each group
  for (int g = warp; g < ng; g += PLAN_WARPS) {
    int e_run = gcnt[g];
    for (int base = 0; base < kc; base += 32) {
      const int ch = base + lane;
      bool any = false;
      for (int p = 0; p < gb && ch < kc; ++p) {
        const int r = gpan[g * MAX_GROUP_PANELS + p];
        if (r >= 0) any |= chunk_kept(mask, r, ch, kb, bpc);
      }
      const unsigned bal = __ballot_sync(0xffffffffu, any);
      if (any) entries[e_run + __popc(bal & lt)] = ch;
      e_run += __popc(bal);
    }
  }
}

__global__ void __launch_bounds__(PLAN_THREADS, 1)
plan_kernel(const uint8_t *__restrict__ mask, int n, int k, int bn, int bk, int32_t *__restrict__ row_ptr,
            int32_t *__restrict__ col_idx, int cap, int32_t *__restrict__ sched) {
  extern __shared__ int plan_smem[];
  plan_body(mask, n, k, bn, bk, row_ptr, col_idx, cap, sched, plan_smem);
}

// Several weights at once: CTA j plans job j.
__global__ void __launch_bounds__(PLAN_THREADS, 1) plan_many_kernel(const __grid_constant__ PackJobs J) {
  extern __shared__ int plan_smem[];
  const PackJob &w = J.job[blockIdx.x];
  plan_body(w.mask, w.n, w.k, w.bn, w.bk, w.row_ptr, w.col_idx, w.cap, w.sched, plan_smem);
}

// Largest i in [0, len) with a[i] <= t, for a[] ascending and a[0] <= t; every lane of the warp
// calls it and gets the answer. Each round splits the range into 32 parts, one load per lane.
__device__ __forceinline__ int warp_last_le(const int32_t *__restrict__ a, int len, int t) {
  const int lane = threadIdx.x & 31;
  int lo = 0, hi = len;  // the answer lies in [lo, hi)
  while (hi - lo > 1) {
    const int step = (hi - lo + 31) >> 5;
    const int i = lo + lane * step;
    const unsigned le = __ballot_sync(0xffffffffu, i < hi && __ldg(a + i) <= t);
    lo += (31 - __clz(le)) * step;  // lane 0 (i = lo) always qualifies
    hi = min(hi, lo + step);
  }
  return lo;
}

constexpr int COPY_THREADS = 128;
constexpr int COPY_WARPS = COPY_THREADS / 32;
constexpr int COPY_CTAS_PER_SM = 6;  // resident at 80 registers a thread: the grid is one wave

// Kept blocks of one weight, one warp per block: blocks t = wi, wi + nw, ... (wi the warp's index
// among nw warps).
__device__ __forceinline__ void copy_body(const uint16_t *__restrict__ W, int n, int k, int bn, int bk,
                                          const int32_t *__restrict__ row_ptr, const int32_t *__restrict__ col_idx,
                                          int cap, uint16_t *__restrict__ blocks, int wi, int nw) {
  const int np = n / bn, lane = threadIdx.x & 31;
  const int nnzb = min(__ldg(row_ptr + np), cap);
  const int lvpr = __ffs(bk / 8) - 1;  // log2 of the 16-byte vectors per block row (bk is a power of 2)
  const int vecs = bn << lvpr;         // 32 .. 512, a multiple of 32
  for (int t = wi; t < nnzb; t += nw) {
    const int r = warp_last_le(row_ptr, np, t), j = __ldg(col_idx + t);
    const uint16_t *src = W + (int64_t)r * bn * k + (int64_t)j * bk;
    int4 *dst = reinterpret_cast<int4 *>(blocks + (int64_t)t * bn * bk);
    for (int v0 = 0; v0 < vecs; v0 += 128) {  // up to four vectors per lane in flight
      int4 val[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int v = v0 + lane + 32 * q;
        if (v < vecs)
          val[q] = __ldg(reinterpret_cast<const int4 *>(src + (int64_t)(v >> lvpr) * k + (v & ((1 << lvpr) - 1)) * 8));
      }
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int v = v0 + lane + 32 * q;
        if (v < vecs) dst[v] = val[q];
      }
    }
  }
}

// Weight-stream tiles of entries e = cta, cta + ncta, ... of one weight (after its plan): the
// group's 256 rows over the entry's 64 columns, row-major, 16-byte vectors; zero where the block
// is removed, where the slot has no panel and beyond column k. Thread i writes vectors
// i + COPY_THREADS * q of the tile: column vector i % 8 of rows i / 8 + 16 q.
__device__ __forceinline__ void stream_body(const uint16_t *__restrict__ W, const uint8_t *__restrict__ mask, int n,
                                            int k, int bn, int bk, const int32_t *__restrict__ sched, int cta,
                                            int ncta) {
  const int kb = k / bk, kc = sched_chunks(k), ng = (n + GROUP_FEATURES - 1) / GROUP_FEATURES;
  if (__ldg(sched + 1) != ng || __ldg(sched + 3) != 0) return;  // not this shape's plan, or blocks overflowed
  const int total = __ldg(sched + 2);
  constexpr int VPR = CHUNK_COLS / 8;                    // 16-byte vectors per tile row
  constexpr int RSTEP = COPY_THREADS / VPR;              // rows between a thread's vectors
  constexpr int PER = GROUP_FEATURES / RSTEP;            // vectors per thread and tile
  static_assert(PER % 8 == 0, "tile rows");
  const int lbn = __ffs(bn) - 1, lbk = __ffs(bk) - 1;  // bn and bk are powers of 2
  const int64_t max_tiles = sched_stream_tiles(ng, kc);
  const int32_t *gent = sched + SCHED_HDR_INTS;
  const int32_t *gpan = sched + sched_gpan_offset_ints(ng);
  const int32_t *ent = sched + sched_entries_offset_ints(ng);
  uint8_t *stream = reinterpret_cast<uint8_t *>(const_cast<int32_t *>(sched)) + sched_stream_offset_bytes(ng, kc);
  const int cv = threadIdx.x % VPR, r0 = threadIdx.x / VPR;
  for (int e = cta; e < total; e += ncta) {
    const int g = warp_last_le(gent, ng, e), ch = __ldg(ent + e);
    if (ch < 0 || ch >= kc || (int64_t)e >= max_tiles) continue;
    int4 *tile = reinterpret_cast<int4 *>(stream + (int64_t)e * stream_tile_bytes());
    const int col = ch * CHUNK_COLS + cv * 8;
    const bool col_ok = col < k;
    const int bc = col >> lbk;
#pragma unroll 1
    for (int h = 0; h < PER; h += 8) {  // eight vectors per thread in flight
      int4 val[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        const int r = r0 + RSTEP * (h + q);
        const int panel = __ldg(gpan + g * MAX_GROUP_PANELS + (r >> lbn));
        // the output feature of group row r (none for an empty slot)
        const int row = panel >= 0 ? (panel << lbn) + (r & (bn - 1)) : -1;
        val[q] = make_int4(0, 0, 0, 0);
        if (row >= 0 && row < n && col_ok && __ldg(mask + (int64_t)panel * kb + bc) != 0)
          val[q] = __ldg(reinterpret_cast<const int4 *>(W + (int64_t)row * k + col));
      }
#pragma unroll
      for (int q = 0; q < 8; ++q) tile[threadIdx.x + COPY_THREADS * (h + q)] = val[q];
    }
  }
}

__global__ void __launch_bounds__(COPY_THREADS, COPY_CTAS_PER_SM)
copy_blocks_kernel(const uint16_t *__restrict__ W, const uint8_t *__restrict__ mask, int n, int k, int bn, int bk,
                   const int32_t *__restrict__ row_ptr, const int32_t *__restrict__ col_idx, int cap,
                   uint16_t *__restrict__ blocks, const int32_t *__restrict__ sched) {
  const int warp = threadIdx.x >> 5;
  if (blocks != nullptr)
    copy_body(W, n, k, bn, bk, row_ptr, col_idx, cap, blocks, blockIdx.x * COPY_WARPS + warp, gridDim.x * COPY_WARPS);
  stream_body(W, mask, n, k, bn, bk, sched, blockIdx.x, gridDim.x);
}

// Several weights at once. The units of job j (kept blocks, one per warp, and stream tiles, one
// per CTA) start where the previous jobs' largest possible counts end (rot_b, rot_t), so that
// the work of all jobs spreads over the whole grid.
__global__ void __launch_bounds__(COPY_THREADS, COPY_CTAS_PER_SM) copy_many_kernel(const __grid_constant__ PackJobs J) {
  const int warp = threadIdx.x >> 5;
  const unsigned ncta = gridDim.x, nw = ncta * COPY_WARPS;
  for (int j = 0; j < J.count; ++j) {
    const PackJob &w = J.job[j];
    if (w.cap > 0 && w.blocks != nullptr) {
      const int wi = (int)((blockIdx.x * COPY_WARPS + warp + (unsigned)w.rot_b) % nw);
      copy_body(w.W, w.n, w.k, w.bn, w.bk, w.row_ptr, w.col_idx, w.cap, w.blocks, wi, (int)nw);
    }
    stream_body(w.W, w.mask, w.n, w.k, w.bn, w.bk, w.sched, (int)((blockIdx.x + (unsigned)w.rot_t) % ncta), (int)ncta);
  }
}

size_t plan_smem_bytes(int n, int k, int bn, int bk) {
  (void)bk;
  const int np = n / bn, ng = (n + GROUP_FEATURES - 1) / GROUP_FEATURES, kc = sched_chunks(k);
  const int W = (kc + 31) / 32;
  size_t words = (size_t)np + 1 + ng + 1 + 33 + np;
  if (grouping_on(np, kc, GROUP_FEATURES / bn)) words += (size_t)np * W + W + np;
  return sizeof(int) * words;
}

cudaError_t launch_pack(const void *W, const uint8_t *mask, int n, int k, int bn, int bk, int32_t *row_ptr,
                        int32_t *col_idx, int cap, void *blocks, int32_t *sched, int num_sms, cudaStream_t s) {
  const size_t smem = plan_smem_bytes(n, k, bn, bk);
  plan_kernel<<<1, PLAN_THREADS, smem, s>>>(mask, n, k, bn, bk, row_ptr, col_idx, cap, sched);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int max_blocks = (n / bn) * (k / bk);
  int grid = (max_blocks + COPY_WARPS - 1) / COPY_WARPS;
  if (grid > num_sms * COPY_CTAS_PER_SM) grid = num_sms * COPY_CTAS_PER_SM;
  if (grid < 1) grid = 1;
  copy_blocks_kernel<<<grid, COPY_THREADS, 0, s>>>(static_cast<const uint16_t *>(W), mask, n, k, bn, bk, row_ptr, col_idx, cap,
                                         static_cast<uint16_t *>(blocks), sched);
  return cudaGetLastError();
}

cudaError_t launch_pack_many(const PackJob *jobs, int count, int num_sms, cudaStream_t s) {
  static bool attr_done[64] = {false};
  for (int first = 0; first < count; first += PACK_MAX_JOBS) {
    PackJobs J;
    J.count = count - first < PACK_MAX_JOBS ? count - first : PACK_MAX_JOBS;
    size_t smem = 0;
    int64_t blocks_max = 0;
    for (int j = 0; j < J.count; ++j) {
      J.job[j] = jobs[first + j];
      const size_t sj = plan_smem_bytes(J.job[j].n, J.job[j].k, J.job[j].bn, J.job[j].bk);
      smem = sj > smem ? sj : smem;
      blocks_max += (int64_t)(J.job[j].n / J.job[j].bn) * (J.job[j].k / J.job[j].bk);
    }
    if (smem > 48 * 1024) {
      int dev = 0;
      cudaGetDevice(&dev);
      if (dev >= 0 && dev < 64 && !attr_done[dev]) {
        cudaError_t e = cudaFuncSetAttribute(plan_many_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             200 * 1024);
        if (e != cudaSuccess) return e;
        attr_done[dev] = true;
      }
    }
    plan_many_kernel<<<J.count, PLAN_THREADS, smem, s>>>(J);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    int64_t grid = (blocks_max + COPY_WARPS - 1) / COPY_WARPS;
    if (grid > (int64_t)num_sms * COPY_CTAS_PER_SM) grid = (int64_t)num_sms * COPY_CTAS_PER_SM;
    if (grid < 1) grid = 1;
    // each job's units start after the previous jobs' largest possible counts (mod the grid)
    const int64_t nw = grid * COPY_WARPS;
    int64_t pb = 0, pt = grid / 2;
    for (int j = 0; j < J.count; ++j) {
      const PackJob &w = J.job[j];
      J.job[j].rot_b = (int)((nw - pb % nw) % nw);
      J.job[j].rot_t = (int)((grid - pt % grid) % grid);
      pb += (int64_t)(w.n / w.bn) * (w.k / w.bk);
      pt += (int64_t)((w.n + GROUP_FEATURES - 1) / GROUP_FEATURES) * sched_chunks(w.k);
    }
    copy_many_kernel<<<(int)grid, COPY_THREADS, 0, s>>>(J);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace lpvit
