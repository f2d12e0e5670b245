/*
 * lpvit.h -- C ABI of liblpvit.so: block-sparse linear layers for LPViT-pruned vision
 * transformers (Xu et al., "LPViT: Low-Power Semi-structured Pruning for Vision
 * Transformers", arXiv 2407.02068), hand-written for NVIDIA GB300 (sm_103a).
 *
 * The operation (Sec. 3.1, block-structured pruning; Sec. 3.3, block-sparse matmul):
 *
 *     Y[m][o] = act( sum_i X[m][i] * W~[o][i] + bias[o] ),
 *     W~[o][i] = W[o][i] if mask[o/bn][i/bk] != 0, else 0,
 *
 * with W stored [n = out features][k = in features] (PyTorch Linear layout), blocks of bn
 * output rows by bk input columns (B_k x B_n in Eq. for P, whose weight is [N in x K out], and the
 * order Table 4 prints, "BK x BN"; bn, bk in {16, 32, 64}, so the
 * square 16x16, 32x32, 64x64 and the paper's 64x32 and 16x32 of Table 2 are all covered),
 * act = identity (lpvit_bsr_linear) or the exact GELU
 * 0.5*y*(1+erf(y/sqrt 2)) (lpvit_bsr_linear_gelu, the DeiT fc1 activation). Only the kept
 * blocks are stored, and removed blocks are never read. The GEMM multiplies, per 256-output group,
 * only the 64-column chunks where the group keeps a block (rows of removed blocks there enter as
 * zeros), so its work follows those group chunks rather than exactly the kept blocks that the
 * power model of Sec. 3.3 (Eq. for P) counts. lpvit_bsr_linear_chain runs a list of such linears
 * (a model's layers, one feeding the next) in one persistent launch.
 *
 * Conventions for every call:
 *  - Array and matrix pointers are DEVICE pointers owned by the caller; the library never
 *    allocates, frees or keeps them. The exceptions live in host memory: nnzb_host, the
 *    lpvit_bsr and lpvit_chain_link structs (and the arrays of them passed to the _many and
 *    _chain calls), which are plain host values holding device pointers, and the host arrays of
 *    lpvit_pack_bsr_many and lpvit_lambda_search. All calls are asynchronous on `stream` (a
 *    cudaStream_t passed as void*, NULL = legacy default stream) unless stated otherwise.
 *  - bf16 means IEEE-754 bfloat16 (raw 16-bit storage); all matrices are row-major.
 *  - A status is returned synchronously for argument errors; CUDA launch errors map to
 *    LPVIT_ERR_CUDA. Errors raised inside a running kernel (a bounded wait that ran out)
 *    are recorded in the workspace and reported by lpvit_check().
 *  - The GPU must be compute capability 10.3 (sm_103a); other devices get
 *    LPVIT_ERR_UNSUPPORTED.
 */
#ifndef LPVIT_H
#define LPVIT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  LPVIT_OK = 0,
  LPVIT_ERR_INVALID_ARG = 1, /* bad shape, null pointer, misaligned pointer or stride      */
  LPVIT_ERR_UNSUPPORTED = 2, /* bn or bk not in {16,32,64}, or not an sm_103 device       */
  LPVIT_ERR_CUDA = 3,        /* a CUDA runtime/driver call failed                          */
  LPVIT_ERR_TIMEOUT = 4,     /* a device-side bounded wait ran out (see lpvit_check)       */
  LPVIT_ERR_WORKSPACE = 5    /* workspace or schedule buffer smaller than required          */
} lpvit_status;

typedef enum { LPVIT_BF16 = 0, LPVIT_F32 = 1 } lpvit_dtype;

/* Block-sparse (BSR) weight, filled by lpvit_pack_bsr. Every pointer is caller-owned device
 * memory of the size stated; the struct itself is a plain host value. A block is bn output rows
 * by bk input columns.
 *   row panel r = output rows [r*bn, (r+1)*bn);  n/bn panels;  block column j = inputs
 *   [j*bk, (j+1)*bk);  k/bk block columns.
 *   row_ptr [n/bn + 1]         int32   exclusive prefix sum of kept blocks per panel
 *   col_idx [nnzb_capacity]    int32   kept block columns of each panel, ascending
 *   blocks  [nnzb_capacity][bn][bk] bf16 kept tiles of W, row-major inside the tile, bits unchanged;
 *                                      may be NULL: the linear reads only `sched`, so the pack then
 *                                      writes row_ptr, col_idx and the work list alone, and the
 *                                      packed weight holds one copy of its kept tiles
 *   sched   [sched_bytes]      bytes   work list for lpvit_bsr_linear (layout private to the
 *                                      library; see lpvit_sched_bytes)
 * nnzb_capacity must be >= the number of kept blocks; (n/bn)*(k/bk) always suffices. */
typedef struct {
  int32_t n, k;
  int32_t bn, bk;
  int32_t nnzb_capacity;
  int32_t *row_ptr;
  int32_t *col_idx;
  void *blocks;
  void *sched;
  size_t sched_bytes;
} lpvit_bsr;

/* Bytes of the `sched` buffer needed for an n x k weight with bn x bk blocks (0 if the shape is
 * invalid). The work list groups the row panels into 256-feature groups (256 / bn panels each,
 * chosen so that the panels of a group keep blocks in overlapping 64-column chunks, or
 * consecutive panels when that gives no fewer chunks) and lists, per group, the chunks where any
 * panel of the group keeps a block (Sec. 3.3: one block matmul per kept block and token tile; a
 * chunk whose blocks are all removed is neither loaded nor multiplied). It also holds a second
 * copy of the kept weights, arranged entry by entry as the GEMM's tensor-core tiles (256 rows x
 * 64 columns, removed blocks as zeros), so that the GEMM reads `sched` and never `blocks`; that
 * copy is sized for a dense weight: 2*64*256 bytes per (group, chunk) plus the list. */
size_t lpvit_sched_bytes(int32_t n, int32_t k, int32_t bn, int32_t bk);

/* Pack W (bf16 [n][k], row-major, 16-byte aligned) under the block mask (uint8 [n/bn][k/bk],
 * nonzero = kept; Sec. 3.1 M_alpha) into bsr->row_ptr / col_idx / blocks and build the work
 * list in bsr->sched. bsr->n, k, bn, bk, nnzb_capacity and all its pointers must be set by the
 * caller. The contents of W inside removed blocks are never read.
 * If nnzb_host is not NULL the call synchronises `stream` and stores the number of kept
 * blocks there. If the mask keeps more blocks than nnzb_capacity, nothing beyond the capacity
 * is written, the work list is marked invalid (linear calls on it then compute nothing and
 * lpvit_check() reports LPVIT_ERR_WORKSPACE), and, when nnzb_host is given, this call returns
 * LPVIT_ERR_WORKSPACE. A capacity of (n/bn)*(k/bk) never overflows.
 * Errors: LPVIT_ERR_INVALID_ARG (shape, null or misaligned pointer), LPVIT_ERR_UNSUPPORTED
 * (bn or bk), LPVIT_ERR_WORKSPACE (sched_bytes too small), LPVIT_ERR_CUDA. */
lpvit_status lpvit_pack_bsr(const void *W, const uint8_t *mask, lpvit_bsr *bsr, int32_t *nnzb_host,
                            void *stream);

/* lpvit_pack_bsr for `count` weights at once, asynchronously on `stream`: W[i] and mask[i] (host
 * arrays of device pointers) are packed into bsr[i] (a host array of count descriptors, set up as
 * for lpvit_pack_bsr). Every job is checked as lpvit_pack_bsr checks its arguments before anything
 * is launched; the first failing check is returned and nothing runs. The jobs travel in the launch
 * parameters (96 per launch), so the call allocates no device memory: all plans run in one launch, one CTA
 * per weight, then all block copies in one more. Results are bit-identical to count calls of
 * lpvit_pack_bsr. There is no kept-block count output; a capacity overflow is reported as for
 * lpvit_pack_bsr (the work list is marked invalid and lpvit_check reports it after a linear).
 * Errors: as lpvit_pack_bsr, and LPVIT_ERR_INVALID_ARG for count < 0 or null arrays. */
lpvit_status lpvit_pack_bsr_many(int32_t count, const void *const *W, const uint8_t *const *mask, lpvit_bsr *bsr,
                                 void *stream);

/* The block mask of Sec. 3.1 ("Block-structured Pruning within layer") from first-order Taylor
 * scores: the neuron score |W . grad W|, a 2D average pooling with the bn x bk block as window
 * and stride, and the bottom-ranked blocks eliminated at pruning ratio `prune_ratio` (alpha).
 *   W       bf16 [n][k] row-major, 16-byte aligned (the weight, as for lpvit_pack_bsr)
 *   G       float32 [n][k] row-major, 16-byte aligned (the gradient of the loss with respect to W)
 *   scores  out: double [n/bn][k/bk], 8-byte aligned: the block scores, in float32 (the
 *           gradient's precision) with a fixed order: each |w * g| rounded to float32, each block
 *           row summed in order, the row sums summed in row order; that total widened to double
 *           and divided by bn*bk. Bit-identical to a plain loop doing the same operations.
 *   mask    out: uint8 [n/bn][k/bk], 1 = kept, 0 = eliminated; it can be passed to lpvit_pack_bsr.
 * Exactly round(alpha * blocks), half away from zero, blocks are eliminated: those ranked lowest,
 * where blocks rank by score and equal scores by linear block index r*(k/bk)+j, the lower first
 * (kept first). W and G must hold finite values. Asynchronous on `stream`; allocates nothing.
 * Errors: LPVIT_ERR_UNSUPPORTED (bn or bk not in {16,32,64}, more than 2^20 blocks),
 * LPVIT_ERR_INVALID_ARG (shape, alpha outside [0, 1], null or misaligned pointer), LPVIT_ERR_CUDA. */
lpvit_status lpvit_taylor_block_mask(const void *W, const float *G, int32_t n, int32_t k, int32_t bn, int32_t bk,
                                     double prune_ratio, double *scores, uint8_t *mask, void *stream);

/* Sec. 3.1 end to end in one call: the Taylor block mask of (W, G) at `prune_ratio` (exactly as
 * lpvit_taylor_block_mask: scores into `scores`, the mask into `mask`) followed by the pack of W
 * under that mask into `bsr` (exactly as lpvit_pack_bsr), all launched on `stream` with no host step
 * between them: the mask passes from the ranking kernel to the pack through `mask` (n/bn x k/bk
 * bytes, which the caller also gets), never through the host. Arguments as for the two calls;
 * nnzb_host as for lpvit_pack_bsr (synchronises `stream` when not NULL).
 * Errors: those of lpvit_taylor_block_mask and lpvit_pack_bsr. */
lpvit_status lpvit_taylor_pack_bsr(const void *W, const float *G, double prune_ratio, double *scores, uint8_t *mask,
                                   lpvit_bsr *bsr, int32_t *nnzb_host, void *stream);

/* The first-order gradient of Sec. 3.1 / 3.5 as the mean of N per-sample gradients:
 * g[e] = (sum_i G[i][e]) / N in float32, the sum in sample order (IEEE float32 additions and
 * division: the precision of the gradients themselves).
 * G float32 [nsamples][count], g float32 [count] (device, 4-byte aligned), 1 <= nsamples <= 1024.
 * This is the gradient lpvit_delta_curve ranks blocks by; pass it to lpvit_taylor_block_mask to
 * get the masks the allocated ratios stand for. Asynchronous on `stream`.
 * Errors: LPVIT_ERR_INVALID_ARG, LPVIT_ERR_CUDA. */
lpvit_status lpvit_mean_gradient(const float *G, int32_t nsamples, int64_t count, float *g, void *stream);

/* Pruning-ratio allocation, Sec. 3.4-3.5. For one layer (weight W, bf16 [n][k], 16-byte aligned)
 * and N per-sample gradients G (float32 [nsamples][n][k], 16-byte aligned), the curve
 *     delta[s] = g . dW_s + 1/2 dW_s^T H dW_s,   s = 0..steps, alpha_s = s / steps,
 * where g = (sum_i G[i]) / N (as lpvit_mean_gradient computes it), dW_s = -W on
 * the blocks (bn rows by bk columns) that the Taylor ranking of Sec. 3.1 under gradient g
 * eliminates at alpha_s (exactly as lpvit_taylor_block_mask would at that ratio) and 0 elsewhere,
 * and H = kappa I + (1/N) sum_i G[i] G[i]^T is the empirical Fisher of Sec. 3.5. It is computed by
 * the incremental update of Eq. update with H in low-rank form (per-block sums of G[i] * W with
 * exact products and float-pair accumulation, about 2^-43 of the block's sum of magnitudes; steps
 * in double; no D x D matrix), delta[0] = 0.
 *   delta     out: double [steps + 1] on the device, 8-byte aligned
 *   workspace device, 256-byte aligned, >= lpvit_delta_curve_workspace_bytes(...) bytes
 * 1 <= nsamples <= 1024, 1 <= steps <= 4096, kappa >= 0 and finite, at most 2^20 blocks.
 * Asynchronous on `stream`; allocates nothing.
 * Errors: LPVIT_ERR_UNSUPPORTED (bn or bk not in {16,32,64}, more than 2^20 blocks),
 * LPVIT_ERR_INVALID_ARG (shape, nsamples, steps, kappa, null or misaligned pointer),
 * LPVIT_ERR_WORKSPACE, LPVIT_ERR_CUDA. */
size_t lpvit_delta_curve_workspace_bytes(int32_t nsamples, int32_t n, int32_t k, int32_t bn, int32_t bk,
                                         int32_t steps);
lpvit_status lpvit_delta_curve(const void *W, const float *G, int32_t nsamples, int32_t n, int32_t k, int32_t bn,
                               int32_t bk, double kappa, int32_t steps, double *delta, void *workspace,
                               size_t ws_bytes, void *stream);

/* The lambda search of Sec. 3.4 (Eq. langrangian2) over per-layer curves; HOST memory, host code,
 * synchronous, no GPU. delta: [layers][steps + 1] (lpvit_delta_curve's output per layer); the
 * distortion of layer i at alpha_s is D_i[s] = delta_i[s]^2 (Eq. obj_f). flops[i] > 0: the layer's
 * dense FLOPs (M N K); power_coef[i] = M N K / (B_n B_k), its power term per unit of (1 - alpha).
 * For a multiplier lambda, layer i takes the largest k such that every slope
 * (D_i[j] - D_i[j-1]) * steps, j = 1..k, is at most lambda + beta * power_coef[i]. Lambda runs
 * over every value at which some layer's k changes (and minus infinity); the result is the
 * smallest such lambda whose FLOPs-remained ratio sum_i (1 - k_i/steps) flops[i] / sum flops is
 * at most flops_ratio (the least pruning that meets the target), else the most pruning.
 *   k_out      out: int32 [layers], alpha_i = k_out[i] / steps
 *   lambda_out, ratio_out   out (may be NULL): the multiplier and the FLOPs-remained ratio
 * Errors: LPVIT_ERR_INVALID_ARG (counts, null pointers, non-finite or non-positive flops,
 * non-finite power_coef or beta, NaN in delta or flops_ratio). */
lpvit_status lpvit_lambda_search(int32_t layers, int32_t steps, const double *delta, const double *flops,
                                 const double *power_coef, double beta, double flops_ratio, int32_t *k_out,
                                 double *lambda_out, double *ratio_out);

/* The non-linear parts of a pre-norm ViT (DeiT) encoder block, so that a whole encoder forward
 * around the block-sparse linears runs in this library (the pruned ViTs of Sec. 4).
 *
 * Residual add + LayerNorm over rows of D features (bf16 [rows][D], row-major, 16-byte aligned):
 *   s = bf16(x + r)  (r may be NULL: s = x),   y = (s - mean) / sqrt(var + eps) * gamma + beta,
 * mean and biased variance over the row in float32; y rounded to bf16 into norm_out, s stored into
 * sum_out when r is given. gamma, beta float32 [D], 16-byte aligned. 8 <= D <= 1024, D % 8 == 0,
 * eps > 0. Asynchronous on `stream`. Errors: LPVIT_ERR_INVALID_ARG, LPVIT_ERR_CUDA. */
lpvit_status lpvit_add_layernorm(const void *x, const void *r, const float *gamma, const float *beta, int64_t rows,
                                 int32_t D, double eps, void *sum_out, void *norm_out, void *stream);

/* Multi-head softmax self-attention per image: qkv bf16 [images * tokens][3 * heads * head_dim]
 * (columns ordered q, k, v, each split into heads of head_dim), out bf16 [images * tokens]
 * [heads * head_dim] = softmax(q k^T / sqrt(head_dim)) v per image and head, heads concatenated.
 * bf16 tensor-core products with fp32 accumulation; the softmax weights are rounded to bf16 for
 * the product with v. head_dim == 64 and 1 <= tokens <= 208 (DeiT: 197) else
 * LPVIT_ERR_UNSUPPORTED; both pointers 16-byte aligned. Asynchronous on `stream`.
 * Errors: LPVIT_ERR_UNSUPPORTED, LPVIT_ERR_INVALID_ARG, LPVIT_ERR_CUDA. */
lpvit_status lpvit_attention(const void *qkv, int64_t images, int32_t tokens, int32_t heads, int32_t head_dim,
                             void *out, void *stream);

/* Bytes of device workspace lpvit_bsr_linear[_gelu] needs for m tokens. The workspace holds
 * scheduler counters, the device error word and, where few token tiles cannot fill the GPU, room
 * for fp32 partial sums of split work units (token counts up to 256 run a single-launch kernel
 * that needs only the counters and the error word; the size asked for does not depend on that).
 * It must be zero-filled once before its first use (cudaMemset); every call leaves its counters
 * at zero again. Calls that may run concurrently must not share a workspace. */
size_t lpvit_workspace_bytes(const lpvit_bsr *bsr, int64_t m);

/* Y = X W~^T + bias for m tokens.
 *   X     bf16 [m][ldx], ldx >= k, ldx % 8 == 0, 16-byte aligned (the first k columns are used)
 *   bias  float32 [n] or NULL (zero bias)
 *   Y     [m][ldy] of y_dtype (bf16, round to nearest even, or float32), ldy >= n;
 *         only columns [0, n) of rows [0, m) are written. X and Y must not overlap.
 *   workspace / ws_bytes: see lpvit_workspace_bytes.
 * Output columns of a panel with no kept block equal bias (or GELU(bias)).
 * m <= 256 (a ViT at batch 1: 197 tokens) runs one launch of plain CTAs, each 128 tokens x 32
 * features of one group over a share of its chunks, a long K cut over the CTAs of a cluster and
 * added in a fixed order; larger m runs the persistent CTA-pair kernel. Both are deterministic:
 * repeated calls give the same bits.
 * Errors: LPVIT_ERR_INVALID_ARG, LPVIT_ERR_UNSUPPORTED, LPVIT_ERR_WORKSPACE, LPVIT_ERR_CUDA. */
lpvit_status lpvit_bsr_linear(const lpvit_bsr *bsr, const void *X, int64_t m, int64_t ldx, const float *bias,
                              void *Y, int64_t ldy, lpvit_dtype y_dtype, void *workspace, size_t ws_bytes,
                              void *stream);

/* As lpvit_bsr_linear, followed by the exact GELU 0.5*y*(1+erf(y/sqrt 2)) (the DeiT MLP fc1). */
lpvit_status lpvit_bsr_linear_gelu(const lpvit_bsr *bsr, const void *X, int64_t m, int64_t ldx,
                                   const float *bias, void *Y, int64_t ldy, lpvit_dtype y_dtype, void *workspace,
                                   size_t ws_bytes, void *stream);

/* Y = round_bf16(round_bf16(act(X W~^T + bias)) + R): lpvit_bsr_linear (gelu == 0) or
 * lpvit_bsr_linear_gelu (gelu == 1) with bf16 output, followed by the residual addition of a
 * pre-norm transformer block (x + sublayer(x), the DeiT blocks whose linears Sec. 4 prunes), done in
 * the GEMM's epilogue instead of a separate pass over the activations. Each sum is formed in float32
 * from the two bf16 values and rounded to nearest even, as a separate bf16 addition would round it.
 *   R    bf16 [m][ldr] device, ldr >= n, ldr % 8 == 0, 16-byte aligned; read only. R may be Y itself
 *        (R == Y and ldr == ldy: Y += the layer, in place); otherwise it must not overlap Y.
 *   gelu 0 or 1.
 * Other arguments, ownership, asynchrony and errors as for lpvit_bsr_linear (y_dtype is bf16).
 * Returns LPVIT_ERR_INVALID_ARG for a null R, a bad ldr or alignment, or a partial overlap of R and Y. */
lpvit_status lpvit_bsr_linear_residual(const lpvit_bsr *bsr, const void *X, int64_t m, int64_t ldx,
                                       const float *bias, int32_t gelu, const void *R, int64_t ldr, void *Y,
                                       int64_t ldy, void *workspace, size_t ws_bytes, void *stream);

/* One linear of a chain: Y = act(X W~^T + bias) with bf16 output, act = GELU when gelu == 1.
 * bsr, X / ldx, bias, Y / ldy and gelu mean what they mean for lpvit_bsr_linear[_gelu]. */
typedef struct {
  const lpvit_bsr *bsr;
  const void *X;
  int64_t ldx;
  const float *bias;
  void *Y;
  int64_t ldy;
  int32_t gelu;
} lpvit_chain_link;

/* Bytes of device workspace lpvit_bsr_linear_chain needs for these links at m tokens (0 for a
 * null or empty list, or a link whose weight shape is invalid): the control block, room for the
 * split-unit partial sums of any link that runs on its own, then the chain's tile counters.
 * Zero-filled once before its first use; every chain call leaves it ready for the next. The same
 * workspace may also serve lpvit_bsr_linear[_gelu] calls on these links' weights at the same m
 * (their scratch lies below the counters); other calls can leave scratch data where the counters
 * are, so give them a workspace of their own. */
size_t lpvit_chain_workspace_bytes(const lpvit_chain_link *links, int32_t count, int64_t m);

/* The linears links[0], links[1], ... links[count-1] over the same m tokens, in that order, as if
 * each were a separate lpvit_bsr_linear (gelu 0) / lpvit_bsr_linear_gelu (gelu 1) call with bf16
 * output on `stream`; the results are bit-identical to those calls. A link may read what earlier
 * links wrote (a model's pruned linears one after another, e.g. fc1 -> fc2, each the block-sparse
 * matmul of Sec. 3.3).
 * Consecutive links run in one persistent launch (up to 48 links per launch): the units of a
 * link follow those of the link before it, and a unit of 256 tokens starts its copies once the
 * previous link has stored every output of those 256 tokens, so one link's last units overlap the
 * next link's first and the launch start and end are paid once per launch, not per link.
 * Row r of every X and Y holds token r. Links share a launch only where their buffers overlap row
 * for row (same leading dimension, a column range of the same rows, e.g. X = the last third of an
 * earlier Y's columns); a link whose buffers overlap an earlier link's otherwise starts a new
 * launch. A link that lpvit_bsr_linear would run on the small-m kernel (m <= 256) or cut into slices
 * (too few 256-token tiles to fill the GPU) runs on its own, as that call would. No Y may overlap
 * a weight, work list or bias of the chain.
 *   workspace / ws_bytes: >= lpvit_chain_workspace_bytes(links, count, m), 256-byte aligned.
 * Every link is checked before anything is launched; nothing runs if one fails.
 * Errors: LPVIT_ERR_INVALID_ARG (count < 0, null links or workspace, gelu not 0 or 1, and the
 * checks of lpvit_bsr_linear for each link), LPVIT_ERR_UNSUPPORTED, LPVIT_ERR_WORKSPACE,
 * LPVIT_ERR_CUDA. count == 0 or m == 0 does nothing and returns LPVIT_OK. */
lpvit_status lpvit_bsr_linear_chain(const lpvit_chain_link *links, int32_t count, int64_t m, void *workspace,
                                    size_t ws_bytes, void *stream);

/* Size of the library-held scratch array used by lpvit_bsr_linear_noalloc (8 MiB). */
#define LPVIT_NOALLOC_SCRATCH_BYTES (8 * 1024 * 1024)

/* As lpvit_bsr_linear (gelu == 0) or lpvit_bsr_linear_gelu (gelu != 0), for callers that cannot
 * allocate device memory where they run this layer: code that has no allocator of its own because
 * another runtime owns all device memory, code recorded while a stream is being captured, or
 * latency-critical paths that must not take the allocator's implicit synchronisation. This entry
 * point has no counterpart in the paper; it only changes who holds the workspace.
 * The workspace is a library-owned device array of LPVIT_NOALLOC_SCRATCH_BYTES that every GPU
 * loading the library keeps until the process exits; the call allocates nothing (no cudaMalloc,
 * cudaFree or allocating library routine). The first call on a device looks up the array's device
 * address (cudaGetSymbolAddress, with that device current) and caches it; make that first call
 * before any stream capture. Each call clears the array's counters on `stream` before launching.
 * All calls share the one array: calls whose kernels may overlap on the GPU (other streams,
 * other host threads) race and give wrong results; serialise them.
 * Errors: as lpvit_bsr_linear, plus LPVIT_ERR_WORKSPACE when lpvit_workspace_bytes(bsr, m)
 * exceeds LPVIT_NOALLOC_SCRATCH_BYTES (large-m calls need well under 1 MiB; small-m calls whose
 * work is split need up to n_tiles * groups * slices * 128 KiB). A device-side timeout is not
 * reported by this entry point (its error word lives in the shared array). */
lpvit_status lpvit_bsr_linear_noalloc(const lpvit_bsr *bsr, const void *X, int64_t m, int64_t ldx,
                                      const float *bias, void *Y, int64_t ldy, lpvit_dtype y_dtype, int gelu,
                                      void *stream);

/* Synchronises `stream`, then reads and clears the error word in `workspace`.
 * Returns LPVIT_OK, LPVIT_ERR_TIMEOUT (a device-side bounded wait ran out; the kernel
 * stopped early and its output is incomplete) or LPVIT_ERR_CUDA. */
lpvit_status lpvit_check(void *workspace, void *stream);

/* Diagnostic of the failure path; it has no counterpart in the paper. Launches, on `stream`, a
 * kernel whose one thread waits on an mbarrier that nothing arrives on, with the bounded wait every
 * role of the GEMM uses: the wait gives up after limit_ns, or after abort_after_ns when that is
 * nonzero (a second thread then raises the CTA's abort flag, as a failing role of the GEMM does).
 * The timeout is recorded in `workspace` (a zero-filled workspace as for lpvit_bsr_linear, 256-byte
 * aligned): the error word, which lpvit_check() then reports as LPVIT_ERR_TIMEOUT and clears, and the
 * microseconds waited, in the 32-bit word at byte offset 12. Nothing else is in flight, so the kernel
 * ends cleanly and the context stays usable.
 * Errors: LPVIT_ERR_INVALID_ARG (null or misaligned workspace, limit_ns 0 or above 10 s,
 * abort_after_ns >= limit_ns), LPVIT_ERR_CUDA (launch failure). */
lpvit_status lpvit_selftest_wait(void *workspace, uint64_t limit_ns, uint64_t abort_after_ns, void *stream);

/* Static English description of a status code. */
const char *lpvit_status_string(lpvit_status status);

#ifdef __cplusplus
}
#endif

#endif /* LPVIT_H */
