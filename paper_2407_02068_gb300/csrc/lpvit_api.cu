// C ABI of liblpvit.so (declared in include/lpvit.h): argument checks, TMA tensor-map encoding,
// work sizing, and launches on the caller's stream. No allocation happens here.
#include <cmath>
#include <cstdint>
#include <cstring>
#include <memory>
#include <mutex>
#include <vector>
#include <cuda.h>
#include <cuda_runtime.h>

#include "lpvit.h"
#include "lpvit_device.cuh"
#include "lpvit_taylor.h"

namespace lpvit {

namespace {

constexpr int MAX_DIM = 65536;
constexpr uint64_t TIMEOUT_NS = 2000000000ull;  // 2 s per wait: far above any legitimate stall

struct DeviceInfo {
  bool queried = false;
  bool supported = false;
  int sms = 0;
};
DeviceInfo g_dev[64];
std::mutex g_mu;

bool device_info(int *sms, lpvit_status *st) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
    *st = LPVIT_ERR_CUDA;
    return false;
  }
  std::lock_guard<std::mutex> lk(g_mu);
  DeviceInfo &d = g_dev[dev];
  if (!d.queried) {
    int major = 0, minor = 0, n = 0;
    if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
      *st = LPVIT_ERR_CUDA;
      return false;
    }
    d.supported = (major == 10 && minor == 3);
    d.sms = n;
    d.queried = true;
  }
  if (!d.supported) {
    *st = LPVIT_ERR_UNSUPPORTED;
    return false;
  }
  *sms = d.sms;
  return true;
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

// Block sides: bn output rows, bk input columns, each 16, 32 or 64.
bool valid_side(int s) { return s == 16 || s == 32 || s == 64; }

bool shape_ok(int n, int k, int bn, int bk) {
  return valid_side(bn) && valid_side(bk) && n > 0 && k > 0 && n <= MAX_DIM && k <= MAX_DIM && n % bn == 0 &&
         k % bk == 0;
}

int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }

// Entries per slice. With at least half as many (token tile, group) units as CTA pairs, a unit
// covers the whole group. Otherwise a group's chunks are cut into slices, whose fp32 partial sums a
// second kernel adds, to bring the unit count towards one per pair, but only while every slice
// keeps at least MIN_SLICE_CHUNKS chunks: below that the partial sums and the reduction launch cost
// more than the extra pairs gain (DeiT batch 1, M = 197: K = 384 and 768 run 1.4-1.8x faster
// unsplit, K = 3072 fastest in four slices).
constexpr int MIN_SLICE_CHUNKS = 12;
int choose_slice(int64_t n_tt, int n_groups, int kc, int pairs) {
  const int64_t units = n_tt * n_groups;
  if (2 * units >= pairs) return kc;
  int64_t nsl = ceil_div(pairs, units);
  const int64_t most = kc / MIN_SLICE_CHUNKS;
  if (nsl > most) nsl = most;
  if (nsl < 1) nsl = 1;
  const int64_t s = ceil_div(kc, nsl);
  return (int)(s < 1 ? 1 : (s > kc ? kc : s));
}

struct WsLayout {
  size_t partials_off, total;
  int S, part_rows;
  bool split;
};

// Workspace: the 256-byte control block, then (split launches only) the fp32 partial sums,
// [token tile][slice][part_rows][GROUP_FEATURES].
WsLayout ws_layout(int64_t m, int n, int k, int sms) {
  WsLayout L;
  const int64_t n_tt = ceil_div(m, TOKENS_PER_TILE);
  const int ng = (int)ceil_div(n, GROUP_FEATURES);
  const int kc = sched_chunks(k);
  L.S = choose_slice(n_tt, ng, kc, sms / 2);
  L.split = L.S < kc;
  L.part_rows = (int)(n_tt == 1 ? m : TOKENS_PER_TILE);
  L.partials_off = sizeof(Control);
  size_t off = L.partials_off;
  if (L.split)
    off += (size_t)n_tt * ng * ceil_div(kc, L.S) * L.part_rows * GROUP_FEATURES * sizeof(float);
  L.total = off;
  return L;
}

lpvit_status cuda_status(cudaError_t e) { return e == cudaSuccess ? LPVIT_OK : LPVIT_ERR_CUDA; }

bool aligned(const void *p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// One linear call, checked and parameterised, ready to launch.
struct Prepared {
  LinearParams P;
  CUtensorMap tmX, tmW;  // the pair kernel's tensor maps (large m)
  WsLayout W;
  int sms = 0;
  bool empty = false;    // m == 0: nothing to do
  bool small = false;    // m <= SMALL_M_MAX: the small-m kernel
};

// The argument checks of a linear call, then its parameter block and tensor maps. Launches nothing.
lpvit_status prepare_linear(const lpvit_bsr *bsr, const void *X, int64_t m, int64_t ldx, const float *bias, void *Y,
                            int64_t ldy, lpvit_dtype y_dtype, void *workspace, size_t ws_bytes, int gelu,
                            const void *R, int64_t ldr, Prepared &pr) {
  if (!bsr) return LPVIT_ERR_INVALID_ARG;
  const int n = bsr->n, k = bsr->k, bn = bsr->bn, bk = bsr->bk;
  if (!valid_side(bn) || !valid_side(bk)) return LPVIT_ERR_UNSUPPORTED;
  if (!shape_ok(n, k, bn, bk)) return LPVIT_ERR_INVALID_ARG;
  if (m < 0) return LPVIT_ERR_INVALID_ARG;
  if (y_dtype != LPVIT_BF16 && y_dtype != LPVIT_F32) return LPVIT_ERR_INVALID_ARG;
  if (m == 0) {
    pr.empty = true;
    return LPVIT_OK;
  }
  if (!X || !Y || !bsr->sched || !workspace) return LPVIT_ERR_INVALID_ARG;
  if (bsr->nnzb_capacity < 0) return LPVIT_ERR_INVALID_ARG;
  if (ldx < k || ldx % 8 != 0 || !aligned(X, 16)) return LPVIT_ERR_INVALID_ARG;
  const size_t ysz = y_dtype == LPVIT_F32 ? 4 : 2;
  if (ldy < n || !aligned(Y, ysz) || !aligned(bsr->sched, 16) || !aligned(workspace, 256))
    return LPVIT_ERR_INVALID_ARG;
  if (bias && !aligned(bias, 4)) return LPVIT_ERR_INVALID_ARG;
  if (m > (int64_t)0x7fffff00) return LPVIT_ERR_INVALID_ARG;
  // X and Y must not overlap
  const uintptr_t y0 = reinterpret_cast<uintptr_t>(Y), y1 = y0 + (size_t)((m - 1) * ldy + n) * ysz;
  {
    const uintptr_t x0 = reinterpret_cast<uintptr_t>(X), x1 = x0 + (size_t)((m - 1) * ldx + k) * 2;
    if (x0 < y1 && y0 < x1) return LPVIT_ERR_INVALID_ARG;
  }
  // the residual: bf16, 16-byte rows like X; either Y itself (in place) or clear of Y
  if (R) {
    if (y_dtype != LPVIT_BF16) return LPVIT_ERR_UNSUPPORTED;
    if (ldr < n || ldr % 8 != 0 || !aligned(R, 16)) return LPVIT_ERR_INVALID_ARG;
    const uintptr_t r0 = reinterpret_cast<uintptr_t>(R), r1 = r0 + (size_t)((m - 1) * ldr + n) * 2;
    const bool in_place = R == Y && ldr == ldy;
    if (!in_place && r0 < y1 && y0 < r1) return LPVIT_ERR_INVALID_ARG;
  }
  if (bsr->sched_bytes < lpvit_sched_bytes(n, k, bn, bk)) return LPVIT_ERR_WORKSPACE;
  lpvit_status st = LPVIT_OK;
  if (!device_info(&pr.sms, &st)) return st;
  pr.W = ws_layout(m, n, k, pr.sms);
  if (ws_bytes < pr.W.total) return LPVIT_ERR_WORKSPACE;
  const int ng = (int)ceil_div(n, GROUP_FEATURES);
  const int kc = sched_chunks(k);
  const int64_t stream_tiles = sched_stream_tiles(ng, kc);
  LinearParams &P = pr.P;
  P.sched = static_cast<const int32_t *>(bsr->sched);
  P.stream_tiles = stream_tiles;
  P.bias = bias;
  P.Y = Y;
  P.ldy = ldy;
  P.m = m;
  P.n = n;
  P.k = k;
  P.bn = bn;
  P.n_tt = (int)ceil_div(m, TOKENS_PER_TILE);
  P.n_groups = ng;
  P.S = pr.W.S;
  P.y_f32 = y_dtype == LPVIT_F32;
  P.gelu = gelu;
  P.y_vec16 = (aligned(Y, 16) && ((size_t)ldy * ysz) % 16 == 0) ? 1 : 0;
  P.y_vec32 = (aligned(Y, 32) && ((size_t)ldy * ysz) % 32 == 0) ? 1 : 0;
  P.bias_vec16 = (bias && aligned(bias, 16)) ? 1 : 0;
  P.R = static_cast<const uint16_t *>(R);
  P.ldr = R ? ldr : 0;
  P.r_vec32 = (R && aligned(R, 32) && ((size_t)ldr * 2) % 32 == 0) ? 1 : 0;
  uint8_t *ws = static_cast<uint8_t *>(workspace);
  P.ctl = reinterpret_cast<Control *>(ws);
  P.partials = reinterpret_cast<float *>(ws + pr.W.partials_off);
  P.part_rows = pr.W.part_rows;
  P.timeout_ns = TIMEOUT_NS;
  P.X = static_cast<const uint16_t *>(X);
  P.ldx = ldx;
  P.wstream = reinterpret_cast<const uint16_t *>(static_cast<const uint8_t *>(bsr->sched) +
                                                 sched_stream_offset_bytes(ng, kc));
  P.kp = 1;
  if (m <= SMALL_M_MAX) {
    pr.small = true;
    return LPVIT_OK;
  }
  EncodeTiledFn enc = encode_fn();
  if (!enc) return LPVIT_ERR_CUDA;

  cuuint32_t es[2] = {1, 1};
  // X: [m rows][k columns], boxes of 64 columns x 128 tokens (one CTA's half of a token tile);
  // rows beyond m and columns beyond k read as zero
  {
    cuuint64_t dims[2] = {(cuuint64_t)k, (cuuint64_t)m};
    cuuint64_t strides[1] = {(cuuint64_t)ldx * 2};
    cuuint32_t box[2] = {(cuuint32_t)CHUNK_COLS, (cuuint32_t)CTA_TOKENS};
    if (enc(&pr.tmX, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(X), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return LPVIT_ERR_INVALID_ARG;
  }
  // the weight stream: tiles of 256 rows x 64 columns, boxes of 128 rows (one CTA's half)
  {
    void *wstream = static_cast<uint8_t *>(bsr->sched) + sched_stream_offset_bytes(ng, kc);
    cuuint64_t dims[2] = {(cuuint64_t)CHUNK_COLS, (cuuint64_t)(stream_tiles * GROUP_FEATURES)};
    cuuint64_t strides[1] = {(cuuint64_t)CHUNK_COLS * 2};
    cuuint32_t box[2] = {(cuuint32_t)CHUNK_COLS, (cuuint32_t)HALF_FEATURES};
    if (enc(&pr.tmW, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, wstream, dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return LPVIT_ERR_INVALID_ARG;
  }
  return LPVIT_OK;
}

// Launches a prepared call: the small-m kernel, or the pair kernel (+ the slice reduction).
lpvit_status launch_prepared(const Prepared &pr, cudaStream_t s) {
  if (pr.empty) return LPVIT_OK;
  const LinearParams &P = pr.P;
  if (pr.small) return cuda_status(launch_linear_small(P, pr.sms, s));
  const int pairs = pr.sms / 2;
  const int kc = sched_chunks(P.k);
  const int64_t units_max = (int64_t)P.n_tt * P.n_groups * ceil_div(kc, P.S);
  const int grid = 2 * (int)(units_max < pairs ? units_max : pairs);
  cudaError_t e = launch_linear(pr.tmX, pr.tmW, P, grid, s);
  if (e != cudaSuccess || !pr.W.split) return cuda_status(e);
  ReduceParams RP;
  RP.sched = P.sched;
  RP.partials = P.partials;
  RP.bias = P.bias;
  RP.Y = P.Y;
  RP.ldy = P.ldy;
  RP.m = P.m;
  RP.n = P.n;
  RP.bn = P.bn;
  RP.n_tt = P.n_tt;
  RP.n_groups = P.n_groups;
  RP.S = P.S;
  RP.part_rows = P.part_rows;
  RP.y_f32 = P.y_f32;
  RP.gelu = P.gelu;
  RP.R = P.R;
  RP.ldr = P.ldr;
  return cuda_status(launch_split_reduce(RP, (int64_t)P.n_tt * P.n_groups * P.part_rows * (GROUP_FEATURES / 8), s));
}

lpvit_status run_linear(const lpvit_bsr *bsr, const void *X, int64_t m, int64_t ldx, const float *bias, void *Y,
                        int64_t ldy, lpvit_dtype y_dtype, void *workspace, size_t ws_bytes, void *stream, int gelu,
                        const void *R = nullptr, int64_t ldr = 0) {
  Prepared pr;
  const lpvit_status st = prepare_linear(bsr, X, m, ldx, bias, Y, ldy, y_dtype, workspace, ws_bytes, gelu, R, ldr, pr);
  if (st != LPVIT_OK) return st;
  return launch_prepared(pr, static_cast<cudaStream_t>(stream));
}

// ---------------------------------------------------------------- chains
// A chain's workspace: the control block and room for the split-unit partial sums of the largest
// of its linears (those run on their own), then the per-(linear, token tile) counters of a launch.
struct ChainWs {
  size_t counters_off, total;
};
size_t align256(size_t x) { return (x + 255) / 256 * 256; }
ChainWs chain_ws_layout(const lpvit_chain_link *links, int32_t count, int64_t m, int sms) {
  size_t most = sizeof(Control);
  for (int32_t i = 0; i < count; ++i) {
    const size_t t = ws_layout(m, links[i].bsr->n, links[i].bsr->k, sms).total;
    if (t > most) most = t;
  }
  ChainWs L;
  L.counters_off = align256(most);
  const int jobs = count < CHAIN_MAX_JOBS ? count : CHAIN_MAX_JOBS;
  L.total = L.counters_off + align256((size_t)jobs * (size_t)ceil_div(m, TOKENS_PER_TILE) * sizeof(uint32_t));
  return L;
}

// A linear joins a chain launch when it runs on the pair kernel without slices.
bool chainable(const Prepared &pr) { return !pr.empty && !pr.small && !pr.W.split && !pr.P.R && !pr.P.y_f32; }

// Row r of two bf16 buffers (base a, row width wa, stride la; base b, wb, lb; in elements) may
// overlap only within token row r: then each linear of a chain touches, in any buffer, only the rows
// of the token tiles it computes, and the tile counters order every access.
bool rows_disjoint_or_aligned(const void *a, int64_t wa, int64_t la, const void *b, int64_t wb, int64_t lb,
                              int64_t m) {
  const intptr_t a0 = reinterpret_cast<intptr_t>(a), b0 = reinterpret_cast<intptr_t>(b);
  const intptr_t a1 = a0 + (intptr_t)((m - 1) * la + wa) * 2, b1 = b0 + (intptr_t)((m - 1) * lb + wb) * 2;
  if (a1 <= b0 || b1 <= a0) return true;
  if (la != lb) return false;
  const intptr_t d = a0 - b0, row = (intptr_t)la * 2;
  return d >= 2 * (intptr_t)wb - row && d + 2 * (intptr_t)wa <= row;
}

// Link j may join a launch that holds links [i, j): every buffer it writes or reads overlaps the
// others' only row for row.
bool joins(const lpvit_chain_link *L, int32_t i, int32_t j, int64_t m) {
  const lpvit_chain_link &c = L[j];
  for (int32_t q = i; q < j; ++q) {
    const lpvit_chain_link &e = L[q];
    if (!rows_disjoint_or_aligned(c.Y, c.bsr->n, c.ldy, e.X, e.bsr->k, e.ldx, m) ||
        !rows_disjoint_or_aligned(c.Y, c.bsr->n, c.ldy, e.Y, e.bsr->n, e.ldy, m) ||
        !rows_disjoint_or_aligned(c.X, c.bsr->k, c.ldx, e.Y, e.bsr->n, e.ldy, m))
      return false;
  }
  return true;
}

// The checks lpvit_pack_bsr applies to one weight.
lpvit_status check_pack_args(const void *W, const uint8_t *mask, const lpvit_bsr *bsr) {
  if (!bsr) return LPVIT_ERR_INVALID_ARG;
  const int n = bsr->n, k = bsr->k, bn = bsr->bn, bk = bsr->bk;
  if (!valid_side(bn) || !valid_side(bk)) return LPVIT_ERR_UNSUPPORTED;
  if (!shape_ok(n, k, bn, bk)) return LPVIT_ERR_INVALID_ARG;
  if (!W || !mask || !bsr->row_ptr || !bsr->sched || bsr->nnzb_capacity < 0) return LPVIT_ERR_INVALID_ARG;
  if (bsr->nnzb_capacity > 0 && !bsr->col_idx) return LPVIT_ERR_INVALID_ARG;  // blocks may be NULL
  if (!aligned(W, 16) || (bsr->blocks && !aligned(bsr->blocks, 16)) || !aligned(bsr->sched, 16) ||
      !aligned(bsr->row_ptr, 4) || (bsr->col_idx && !aligned(bsr->col_idx, 4)))
    return LPVIT_ERR_INVALID_ARG;
  if (bsr->sched_bytes < lpvit_sched_bytes(n, k, bn, bk)) return LPVIT_ERR_WORKSPACE;
  return LPVIT_OK;
}

}  // namespace
}  // namespace lpvit

using namespace lpvit;

extern "C" {

size_t lpvit_sched_bytes(int32_t n, int32_t k, int32_t bn, int32_t bk) {
  if (!shape_ok(n, k, bn, bk)) return 0;
  const int ng = (int)ceil_div(n, GROUP_FEATURES);
  const int kc = sched_chunks(k);
  return (size_t)sched_stream_offset_bytes(ng, kc) + (size_t)sched_stream_tiles(ng, kc) * stream_tile_bytes();
}


lpvit_status lpvit_pack_bsr(const void *W, const uint8_t *mask, lpvit_bsr *bsr, int32_t *nnzb_host, void *stream) {
  const lpvit_status chk = check_pack_args(W, mask, bsr);
  if (chk != LPVIT_OK) return chk;
  const int n = bsr->n, k = bsr->k, bn = bsr->bn, bk = bsr->bk;
  int sms = 0;
  lpvit_status st = LPVIT_OK;
  if (!device_info(&sms, &st)) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e = launch_pack(W, mask, n, k, bn, bk, bsr->row_ptr, bsr->col_idx, bsr->nnzb_capacity, bsr->blocks,
                              static_cast<int32_t *>(bsr->sched), sms, s);
  if (e != cudaSuccess) return LPVIT_ERR_CUDA;
  if (nnzb_host) {
    int32_t v = 0;
    e = cudaMemcpyAsync(&v, bsr->row_ptr + n / bn, sizeof(v), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return LPVIT_ERR_CUDA;
    *nnzb_host = v;
    if (v > bsr->nnzb_capacity) return LPVIT_ERR_WORKSPACE;
  }
  return LPVIT_OK;
}

lpvit_status lpvit_taylor_pack_bsr(const void *W, const float *G, double prune_ratio, double *scores, uint8_t *mask,
                                   lpvit_bsr *bsr, int32_t *nnzb_host, void *stream) {
  const lpvit_status chk = check_pack_args(W, mask, bsr);
  if (chk != LPVIT_OK) return chk;
  const int n = bsr->n, k = bsr->k, bn = bsr->bn, bk = bsr->bk;
  if (!(prune_ratio >= 0.0 && prune_ratio <= 1.0)) return LPVIT_ERR_INVALID_ARG;  // also rejects NaN
  if (!G || !scores || !aligned(G, 16) || !aligned(scores, 8)) return LPVIT_ERR_INVALID_ARG;
  const int64_t total = (int64_t)(n / bn) * (k / bk);
  if (total > (int64_t)1 << 20) return LPVIT_ERR_UNSUPPORTED;
  int sms = 0;
  lpvit_status st = LPVIT_OK;
  if (!device_info(&sms, &st)) return st;
  // eliminated = round(alpha * blocks), half away from zero (as lpvit_taylor_block_mask)
  const int64_t keep = total - (int64_t)floor(prune_ratio * (double)total + 0.5);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (launch_block_scores(static_cast<const uint16_t *>(W), G, n, k, bn, bk, scores, s) != cudaSuccess ||
      launch_block_rank(scores, total, keep, mask, nullptr, s) != cudaSuccess)
    return LPVIT_ERR_CUDA;
  cudaError_t e = launch_pack(W, mask, n, k, bn, bk, bsr->row_ptr, bsr->col_idx, bsr->nnzb_capacity, bsr->blocks,
                              static_cast<int32_t *>(bsr->sched), sms, s);
  if (e != cudaSuccess) return LPVIT_ERR_CUDA;
  if (nnzb_host) {
    int32_t v = 0;
    e = cudaMemcpyAsync(&v, bsr->row_ptr + n / bn, sizeof(v), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return LPVIT_ERR_CUDA;
    *nnzb_host = v;
    if (v > bsr->nnzb_capacity) return LPVIT_ERR_WORKSPACE;
  }
  return LPVIT_OK;
}

lpvit_status lpvit_pack_bsr_many(int32_t count, const void *const *W, const uint8_t *const *mask, lpvit_bsr *bsr,
                                 void *stream) {
  if (count < 0) return LPVIT_ERR_INVALID_ARG;
  if (count == 0) return LPVIT_OK;
  if (!W || !mask || !bsr) return LPVIT_ERR_INVALID_ARG;
  for (int32_t i = 0; i < count; ++i) {
    const lpvit_status chk = check_pack_args(W[i], mask[i], &bsr[i]);
    if (chk != LPVIT_OK) return chk;
  }
  int sms = 0;
  lpvit_status st = LPVIT_OK;
  if (!device_info(&sms, &st)) return st;
  std::vector<PackJob> jobs((size_t)count);
  for (int32_t i = 0; i < count; ++i) {
    PackJob &j = jobs[(size_t)i];
    j.W = static_cast<const uint16_t *>(W[i]);
    j.mask = mask[i];
    j.row_ptr = bsr[i].row_ptr;
    j.col_idx = bsr[i].col_idx;
    j.blocks = static_cast<uint16_t *>(bsr[i].blocks);
    j.sched = static_cast<int32_t *>(bsr[i].sched);
    j.n = bsr[i].n;
    j.k = bsr[i].k;
    j.bn = bsr[i].bn;
    j.bk = bsr[i].bk;
    j.cap = bsr[i].nnzb_capacity;
  }
  return cuda_status(launch_pack_many(jobs.data(), count, sms, static_cast<cudaStream_t>(stream)));
}

size_t lpvit_workspace_bytes(const lpvit_bsr *bsr, int64_t m) {
  if (!bsr || !shape_ok(bsr->n, bsr->k, bsr->bn, bsr->bk) || m < 0) return 0;
  int sms = 0;
  lpvit_status st = LPVIT_OK;
  if (!device_info(&sms, &st)) sms = 152;  // sizing only; the call itself reports the device error
  return ws_layout(m > 0 ? m : 1, bsr->n, bsr->k, sms).total;
}

lpvit_status lpvit_bsr_linear(const lpvit_bsr *bsr, const void *X, int64_t m, int64_t ldx, const float *bias,
                              void *Y, int64_t ldy, lpvit_dtype y_dtype, void *workspace, size_t ws_bytes,
                              void *stream) {
  return run_linear(bsr, X, m, ldx, bias, Y, ldy, y_dtype, workspace, ws_bytes, stream, 0);
}

lpvit_status lpvit_bsr_linear_gelu(const lpvit_bsr *bsr, const void *X, int64_t m, int64_t ldx,
                                   const float *bias, void *Y, int64_t ldy, lpvit_dtype y_dtype, void *workspace,
                                   size_t ws_bytes, void *stream) {
  return run_linear(bsr, X, m, ldx, bias, Y, ldy, y_dtype, workspace, ws_bytes, stream, 1);
}

lpvit_status lpvit_bsr_linear_residual(const lpvit_bsr *bsr, const void *X, int64_t m, int64_t ldx,
                                       const float *bias, int32_t gelu, const void *R, int64_t ldr, void *Y,
                                       int64_t ldy, void *workspace, size_t ws_bytes, void *stream) {
  if (!R || (gelu != 0 && gelu != 1)) return LPVIT_ERR_INVALID_ARG;
  return run_linear(bsr, X, m, ldx, bias, Y, ldy, LPVIT_BF16, workspace, ws_bytes, stream, gelu, R, ldr);
}

size_t lpvit_chain_workspace_bytes(const lpvit_chain_link *links, int32_t count, int64_t m) {
  if (!links || count <= 0 || m < 0) return 0;
  for (int32_t i = 0; i < count; ++i)
    if (!links[i].bsr || !shape_ok(links[i].bsr->n, links[i].bsr->k, links[i].bsr->bn, links[i].bsr->bk)) return 0;
  int sms = 0;
  lpvit_status st = LPVIT_OK;
  if (!device_info(&sms, &st)) sms = 152;  // sizing only; the call itself reports the device error
  return chain_ws_layout(links, count, m > 0 ? m : 1, sms).total;
}

lpvit_status lpvit_bsr_linear_chain(const lpvit_chain_link *links, int32_t count, int64_t m, void *workspace,
                                    size_t ws_bytes, void *stream) {
  if (count < 0 || m < 0) return LPVIT_ERR_INVALID_ARG;
  if (count == 0 || m == 0) return LPVIT_OK;
  if (!links || !workspace || !aligned(workspace, 256)) return LPVIT_ERR_INVALID_ARG;
  // every link is checked before anything is launched
  for (int32_t i = 0; i < count; ++i)
    if (!links[i].bsr || (links[i].gelu != 0 && links[i].gelu != 1)) return LPVIT_ERR_INVALID_ARG;
  std::vector<Prepared> pr((size_t)count);
  for (int32_t i = 0; i < count; ++i) {
    const lpvit_chain_link &c = links[i];
    const lpvit_status st = prepare_linear(c.bsr, c.X, m, c.ldx, c.bias, c.Y, c.ldy, LPVIT_BF16, workspace, ws_bytes,
                                           c.gelu, nullptr, 0, pr[(size_t)i]);
    if (st != LPVIT_OK) return st;
  }
  const ChainWs CW = chain_ws_layout(links, count, m, pr[0].sms);
  if (ws_bytes < CW.total) return LPVIT_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int n_tt = (int)ceil_div(m, TOKENS_PER_TILE);
  std::unique_ptr<ChainParams> C(new ChainParams());
  for (int32_t i = 0; i < count;) {
    // the longest run from link i that one launch takes
    int32_t j = i + 1;
    uint64_t units = chainable(pr[(size_t)i]) ? (uint64_t)n_tt * pr[(size_t)i].P.n_groups : 0;
    if (chainable(pr[(size_t)i]))
      while (j < count && j - i < CHAIN_MAX_JOBS && chainable(pr[(size_t)j]) && joins(links, i, j, m) &&
             units + (uint64_t)n_tt * pr[(size_t)j].P.n_groups <= 0x7fffffffull) {
        units += (uint64_t)n_tt * pr[(size_t)j].P.n_groups;
        ++j;
      }
    if (j - i == 1) {  // a run of one: the linear's own launch
      const lpvit_status st = launch_prepared(pr[(size_t)i], s);
      if (st != LPVIT_OK) return st;
      i = j;
      continue;
    }
    uint32_t u0 = 0;
    for (int32_t q = i; q < j; ++q) {
      ChainJob &J = C->job[q - i];
      const Prepared &p = pr[(size_t)q];
      J.tmX = p.tmX;
      J.tmW = p.tmW;
      J.P = p.P;
      J.unit0 = u0;
      J.units = (uint32_t)n_tt * (uint32_t)p.P.n_groups;
      u0 += J.units;
    }
    C->tile_done = reinterpret_cast<uint32_t *>(static_cast<uint8_t *>(workspace) + CW.counters_off);
    C->total_units = u0;
    C->njobs = j - i;
    C->n_tt = n_tt;
    const int pairs = pr[0].sms / 2;
    const int grid = 2 * (int)((int64_t)u0 < pairs ? (int64_t)u0 : pairs);
    const cudaError_t e = launch_linear_chain(*C, grid, s);
    if (e != cudaSuccess) return LPVIT_ERR_CUDA;
    i = j;
  }
  return LPVIT_OK;
}

lpvit_status lpvit_check(void *workspace, void *stream) {
  if (!workspace) return LPVIT_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaStreamSynchronize(s) != cudaSuccess) return LPVIT_ERR_CUDA;
  Control *ctl = static_cast<Control *>(workspace);
  unsigned int err = 0;
  if (cudaMemcpy(&err, &ctl->err, sizeof(err), cudaMemcpyDeviceToHost) != cudaSuccess) return LPVIT_ERR_CUDA;
  if (err) {
    if (cudaMemset(&ctl->err, 0, sizeof(err)) != cudaSuccess) return LPVIT_ERR_CUDA;
    if (err & (ERR_SCHED_OVERFLOW | ERR_BAD_SCHED)) return LPVIT_ERR_WORKSPACE;
    return LPVIT_ERR_TIMEOUT;
  }
  return LPVIT_OK;
}

const char *lpvit_status_string(lpvit_status status) {
  switch (status) {
    case LPVIT_OK: return "ok";
    case LPVIT_ERR_INVALID_ARG: return "invalid argument (shape, null or misaligned pointer or stride)";
    case LPVIT_ERR_UNSUPPORTED: return "unsupported (a block side not 16/32/64, or device is not sm_103)";
    case LPVIT_ERR_CUDA: return "CUDA runtime or driver error";
    case LPVIT_ERR_TIMEOUT: return "a device-side bounded wait ran out; the output is incomplete";
    case LPVIT_ERR_WORKSPACE: return "workspace, schedule buffer or block capacity too small";
  }
  return "unknown status";
}

}  // extern "C"
