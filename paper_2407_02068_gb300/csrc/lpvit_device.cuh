// Device-side building blocks for sm_103a: mbarriers with bounded waits, TMA (tensor and bulk),
// tcgen05 (TMEM allocation, MMA from shared memory, TMEM loads) and the shared-memory matrix /
// instruction descriptors they take. All inline PTX, no libraries.
#pragma once
#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

namespace lpvit {

// Layout of the work list ("sched") shared by the pack and the GEMM, for blocks of bn output rows
// by bk input columns. The GEMM covers the weight in tiles of GROUP_FEATURES output features by
// CHUNK_COLS input columns (one pipeline stage of MMAs), and skips the tiles whose blocks are all
// removed.
// header (16 int32): [0] nnzb, [1] n_groups, [2] total entries, [3] overflow flag, [4] n, [5] k,
// [6] bn, [7] bk, [8] layout version (SCHED_VERSION)
// then gent_ptr[n_groups + 1] (int32, entries of group g are [gent_ptr[g], gent_ptr[g+1]))
// then gpan[n_groups][MAX_GROUP_PANELS] (int32): the row panel in slot p of group g, or -1. A group
// is GROUP_FEATURES / bn row panels, not necessarily consecutive: the plan picks panels whose kept
// chunks overlap, so that a group has fewer entries; group row r is panel gpan[g][r / bn], row
// r % bn, i.e. output feature gpan[g][r / bn] * bn + r % bn.
// then entries, one int32 each: the chunk index c (input columns [c * CHUNK_COLS, (c + 1) *
// CHUNK_COLS)) of a tile of the group holding at least one kept block; entry e's tile in the
// weight stream is tile e;
// then, at sched_stream_offset_bytes (1024-byte aligned), the weight stream: per entry a tile of
// GROUP_FEATURES rows of CHUNK_COLS bf16, row-major (128-byte rows), row r = group row r:
// W[feature][c * CHUNK_COLS + col] where its block is kept, zero where it is removed, where the
// slot has no panel and beyond column k. The GEMM's tensor copies load each 128-row half with the
// 128-byte swizzle its MMA descriptors read.
constexpr int SCHED_HDR_INTS = 16;
constexpr int SCHED_VERSION = 2;
constexpr int GROUP_FEATURES = 256;   // output features of one work unit (the pair MMA's N)
constexpr int HALF_FEATURES = GROUP_FEATURES / 2;  // weight rows one CTA of the pair stages
constexpr int MAX_GROUP_PANELS = GROUP_FEATURES / 16;
constexpr int CHUNK_COLS = 64;        // input columns per stage: four 16-wide MMA k steps
constexpr int TOKENS_PER_TILE = 256;  // tokens of one work unit (the pair MMA's M)
constexpr int CTA_TOKENS = TOKENS_PER_TILE / 2;

__host__ __device__ inline int sched_chunks(int k) { return (k + CHUNK_COLS - 1) / CHUNK_COLS; }
__host__ __device__ inline int sched_gent_offset_ints() { return SCHED_HDR_INTS; }
__host__ __device__ inline int64_t sched_gpan_offset_ints(int n_groups) { return (int64_t)SCHED_HDR_INTS + n_groups + 1; }
__host__ __device__ inline int64_t sched_entries_offset_ints(int n_groups) {
  return (sched_gpan_offset_ints(n_groups) + (int64_t)n_groups * MAX_GROUP_PANELS + 3) / 4 * 4;  // 16-byte aligned
}
__host__ __device__ inline int64_t sched_stream_offset_bytes(int n_groups, int kc) {
  const int64_t end = 4 * (sched_entries_offset_ints(n_groups) + (int64_t)n_groups * kc);
  return (end + 1023) / 1024 * 1024;
}
__host__ __device__ constexpr int stream_tile_bytes() { return GROUP_FEATURES * CHUNK_COLS * 2; }
// Tiles the stream region holds: one per group and chunk (the most entries there can be).
__host__ __device__ inline int64_t sched_stream_tiles(int n_groups, int kc) { return (int64_t)n_groups * kc; }
static_assert(MAX_GROUP_PANELS <= 16, "a group's slot mask fits 16 bits");

// Workspace control block (first 256 bytes of the caller's workspace).
struct Control {
  unsigned int next_unit;   // dynamic scheduler: next unit to hand out
  unsigned int done_ctas;   // CTAs that found the queue empty; the last one resets both
  unsigned int err;         // device error word (bit set per failing wait site), read by lpvit_check
  unsigned int err_detail;
  unsigned int chain_ctas;  // chain launches: CTAs that have finished; the last one resets the tile counters
  unsigned int pad[59];
};
static_assert(sizeof(Control) == 256, "control block is 256 bytes");

// Parameter block of the linear kernel (host fills it, the kernel reads it by value).
struct LinearParams {
  const int32_t *sched;    // work list (header, gent_ptr, gpan, entries)
  int64_t stream_tiles;    // tiles the stream region holds (bound on every entry's tile)
  const float *bias;       // [n] or nullptr
  void *Y;
  int64_t ldy;
  int64_t m;
  int n, k;
  int bn;                  // block height: a group holds GROUP_FEATURES / bn row panels
  int n_tt, n_groups, S;   // token tiles, groups, max entries per slice
  int y_f32, gelu;
  int y_vec16;             // output rows may take 16-byte stores (Y 16-byte aligned, ldy * size % 16 == 0)
  int y_vec32;             // ... and 32-byte stores (Y 32-byte aligned, ldy * size % 32 == 0)
  int bias_vec16;          // bias is 16-byte aligned
  const uint16_t *R;       // bf16 residual [m][ldr] added after rounding (bf16 output only), or nullptr
  int64_t ldr;
  int r_vec32;             // residual rows may take 32-byte loads (else 16-byte ones)
  Control *ctl;
  float *partials;         // split units: [slice][part_rows][GROUP_FEATURES] fp32 partial sums
  int part_rows;           // token rows of one partial tile: min(m, TOKENS_PER_TILE)
  uint64_t timeout_ns;     // limit of every device-side wait
  // read by the small-m kernel only (the pair kernel reaches X and the stream through tensor maps)
  const uint16_t *X;       // bf16 [m][ldx]
  int64_t ldx;
  const uint16_t *wstream; // the work list's weight stream
  int kp;                  // K parts per (group, row slice, token tile): the CTAs of one cluster
};

// Parameter block of the split-slice reduction (after the linear kernel, same stream).
struct ReduceParams {
  const int32_t *sched;
  const float *partials;
  const float *bias;
  void *Y;
  int64_t ldy;
  int64_t m;
  int n, bn;
  int n_tt, n_groups, S;
  int part_rows;
  int y_f32, gelu;
  const uint16_t *R;
  int64_t ldr;
};

enum ErrBits : unsigned int {
  ERR_PRODUCER_EMPTY = 1u << 0,
  ERR_PRODUCER_UNIT = 1u << 1,
  ERR_MMA_FULL = 1u << 2,
  ERR_MMA_ACC = 1u << 3,
  ERR_MMA_UNIT = 1u << 4,
  ERR_EPI_ACC = 1u << 5,
  ERR_EPI_UNIT = 1u << 6,
  ERR_DRAIN = 1u << 7,
  ERR_SCHED_OVERFLOW = 1u << 8,
  ERR_BAD_SCHED = 1u << 9,
  ERR_CHAIN_WAIT = 1u << 10,
};

// Launchers (host side, defined next to their kernels).
cudaError_t launch_pack(const void *W, const uint8_t *mask, int n, int k, int bn, int bk, int32_t *row_ptr,
                        int32_t *col_idx, int cap, void *blocks, int32_t *sched, int num_sms, cudaStream_t s);

// One weight of a batched pack; the whole table travels in the kernel parameters.
struct PackJob {
  const uint16_t *W;
  const uint8_t *mask;
  int32_t *row_ptr;
  int32_t *col_idx;
  uint16_t *blocks;
  int32_t *sched;
  int n, k, bn, bk, cap;
  int rot_b, rot_t;  // set by launch_pack_many: where the job's block and tile units start
};
constexpr int PACK_MAX_JOBS = 96;  // jobs per launch (6 KB of parameters)
struct PackJobs {
  int count;
  PackJob job[PACK_MAX_JOBS];
};
cudaError_t launch_pack_many(const PackJob *jobs, int count, int num_sms, cudaStream_t s);
// grid = 2 * pairs (clusters of two CTAs); a split launch is followed by the reduction.
cudaError_t launch_linear(const CUtensorMap &tmX, const CUtensorMap &tmW, const LinearParams &P, int grid,
                          cudaStream_t s);
cudaError_t launch_split_reduce(const ReduceParams &R, int64_t threads, cudaStream_t s);
// A chain: consecutive linears over the same m tokens in one persistent launch of the pair kernel.
// Linear j's units follow linear j - 1's in the unit order; a unit of linear j > 0 loads its X tile
// only once every unit of linear j - 1 for the same token tile has stored its outputs (both CTAs of
// each of its n_groups units: 2 n_groups arrivals on tile_done[j - 1][tile]). Only linears whose
// groups are not cut into slices, with bf16 output and no residual, are chained.
struct ChainJob {
  CUtensorMap tmX;   // this linear's input (any earlier linear's output, or the chain's input)
  CUtensorMap tmW;   // its weight stream
  LinearParams P;
  uint32_t unit0;    // index of its first unit in the chain's unit order
  uint32_t units;    // n_tt * n_groups
};
constexpr int CHAIN_MAX_JOBS = 48;  // linears per launch (the whole table travels in the parameters)
struct ChainParams {
  ChainJob job[CHAIN_MAX_JOBS];
  uint32_t *tile_done;   // [njobs][n_tt] stored-unit arrivals per (linear, token tile); zero at entry
  uint32_t total_units;
  int njobs, n_tt;
};
static_assert(sizeof(ChainParams) <= 32764, "kernel parameter space");
cudaError_t launch_linear_chain(const ChainParams &C, int grid, cudaStream_t s);
// Token counts up to SMALL_M_MAX take the small-m kernel (one launch, no workspace beyond the
// control block); it sets P.kp itself.
constexpr int SMALL_M_MAX = 256;
cudaError_t launch_linear_small(LinearParams P, int num_sms, cudaStream_t s);

__device__ __forceinline__ uint32_t smem_u32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ uint32_t elect_one() {
  uint32_t pred = 0;
  asm volatile("{.reg .b32 rx; .reg .pred px; elect.sync rx|px, 0xffffffff; selp.u32 %0, 1, 0, px;}" : "=r"(pred));
  return pred;
}

// ------------------------------------------------------------------ mbarrier
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" :: "r"(bar), "r"(count));
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" :: "r"(bar) : "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" :: "r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile("{.reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p;}"
               : "=r"(ok) : "r"(bar), "r"(parity) : "memory");
  return ok != 0;
}

// Bounded wait: returns false after `limit_ns` without completion, or as soon as another role of
// this CTA has raised the abort flag. Never spins forever.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, const volatile int *abort_flag,
                                          uint64_t limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (;;) {
#pragma unroll 1
    for (int i = 0; i < 32; ++i)
      if (mbar_try_wait(bar, parity)) return true;
    if (*abort_flag) return false;
    if (globaltimer_ns() - t0 > limit_ns) return false;
  }
}

// ------------------------------------------------------------------ TMA
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *map, int32_t x, int32_t y, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];"
      :: "r"(dst), "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar) : "memory");
}
// Untiled bulk copy global -> shared: both addresses 16-byte aligned, bytes a multiple of 16.
__device__ __forceinline__ void bulk_load(uint32_t dst, const void *src, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
               :: "r"(dst), "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(bar) : "memory");
}
__device__ __forceinline__ void prefetch_tensormap(const CUtensorMap *map) {
  asm volatile("prefetch.tensormap [%0];" :: "l"(reinterpret_cast<uint64_t>(map)) : "memory");
}
__device__ __forceinline__ void fence_proxy_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// 16-byte asynchronous copy global -> shared; src_bytes < 16 fills the rest with zeros (0: no read).
__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src, uint32_t src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" :: "r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" :: "n"(N) : "memory"); }
// Byte offset of 16-byte piece j of row r in a K-major tile of 128-byte rows stored with the
// 128-byte swizzle (tile base 1024-byte aligned), the layout smem_desc<128> describes.
__device__ __forceinline__ uint32_t sw_off(int r, int j) { return (uint32_t)(r * 128 + ((j ^ (r & 7)) << 4)); }

// ------------------------------------------------------------------ tcgen05
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" :: "r"(dst_smem), "r"(ncols));
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" :: "r"(taddr), "r"(ncols));
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" :: "r"(bar) : "memory");
}

// ------------------------------------------------------------------ CTA pairs (cluster of 2)
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// The cluster address of this CTA's shared-memory location `a` in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t mapa_rank(uint32_t a, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(rank));
  return r;
}
// Arrive on an mbarrier of either CTA of the cluster (release at cluster scope: earlier writes of
// this thread, to either CTA's shared memory, are visible to the waiter).
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" :: "r"(cluster_addr) : "memory");
}
__device__ __forceinline__ void st_cluster_v4(uint32_t cluster_addr, int4 v) {
  asm volatile("st.shared::cluster.v4.b32 [%0], {%1, %2, %3, %4};" :: "r"(cluster_addr), "r"(v.x), "r"(v.y), "r"(v.z),
               "r"(v.w) : "memory");
}
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// Tensor copy into this CTA's shared memory whose completion is counted on an mbarrier of either
// CTA of the pair (cluster address).
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const CUtensorMap *map, int32_t x, int32_t y,
                                                 uint32_t bar_cluster) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.cta_group::2 "
      "[%0], [%1, {%2, %3}], [%4];"
      :: "r"(dst), "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar_cluster) : "memory");
}
// TMEM allocation for the pair: one warp of each CTA executes it, both get the same columns.
__device__ __forceinline__ void tmem_alloc_pair(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" :: "r"(dst_smem), "r"(ncols));
}
__device__ __forceinline__ void tmem_relinquish_pair() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;");
}
__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" :: "r"(taddr), "r"(ncols));
}
// Arrive once on the mbarrier at shared-memory offset `bar` of every CTA in `mask` when this
// thread's earlier pair MMAs complete.
__device__ __forceinline__ void tc_commit_pair(uint32_t bar, uint16_t mask) {
  asm volatile("tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;"
               :: "r"(bar), "h"(mask) : "memory");
}
// D[256 x N] (+)= A[256 x 16] * B[N x 16]^T over the CTA pair: A rows 0-127 from this CTA's shared
// memory, 128-255 from the peer's (same offset); B rows 0 .. N/2 - 1 from this CTA, the rest from
// the peer; D rows 0-127 in this CTA's TMEM, 128-255 in the peer's. Issued by the leader alone.
__device__ __forceinline__ void umma_f16_pair(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                              uint32_t accumulate) {
  asm volatile("{.reg .pred p; setp.ne.b32 p, %4, 0;\n"
               "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;}\n"
               :: "r"(d_tmem), "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate));
}

// Shared-memory matrix descriptor for a K-major operand tile whose rows are `row_bytes`
// (32, 64 or 128) long and stored with the matching TMA swizzle; 8-row atoms are contiguous.
template <int ROW_BYTES>
__device__ __forceinline__ uint64_t smem_desc(uint32_t saddr) {
  static_assert(ROW_BYTES == 32 || ROW_BYTES == 64 || ROW_BYTES == 128, "row bytes");
  constexpr uint64_t layout = ROW_BYTES == 128 ? 2 : (ROW_BYTES == 64 ? 4 : 6);  // SW128 / SW64 / SW32
  constexpr uint64_t sbo = 8 * ROW_BYTES;                                     // bytes between 8-row atoms
  return (uint64_t)((saddr & 0x3FFFF) >> 4) | ((uint64_t)1 << 16) | ((sbo >> 4) << 32) | ((uint64_t)1 << 46) |
         (layout << 61);
}

// Instruction descriptor, kind::f16: bf16 x bf16 -> fp32, both operands K-major.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

// MMA D[M x N] (+)= A[M x 16] * B[N x 16]^T, A and B K-major in shared memory (descriptors), D
// fp32 in TMEM (row i in lane i, column j in column j); `accumulate` = 0 overwrites D. One thread
// issues it; the caller computes the warp-uniform operands with the whole warp.
__device__ __forceinline__ void umma_f16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                         uint32_t accumulate) {
  asm volatile("{.reg .pred p; setp.ne.b32 p, %4, 0;\n"
               "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;}\n"
               :: "r"(d_tmem), "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate));
}

// TMEM -> registers: 32 lanes x 32 consecutive 32-bit columns (one lane per thread).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

}  // namespace lpvit
