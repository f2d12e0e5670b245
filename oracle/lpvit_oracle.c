/*
 * Plain, slow CPU oracle for the block-sparse linear layer of LPViT (arXiv 2407.02068).
 *
 * TEST INFRASTRUCTURE ONLY. Nothing in the product path may include, link or call this file:
 * only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline / reference arm use it.
 * It shares no code, header, table or helper with the CUDA library.
 *
 * What it computes (all arithmetic in IEEE double precision):
 *
 *  - Block-structured pruning mask, Sec. 3.1 ("Block-structured Pruning within layer"):
 *      W~[i][j] = W[i][j] (.) M[ceil(i/B_h)][ceil(j/B_w)]
 *    The paper indexes blocks 1-based with a ceiling; with 0-based indices the block of
 *    element (i, j) is (floor(i/bn), floor(j/bk)), a block being bn output rows by bk input
 *    columns. Eq. for P writes the weight as [N inputs x K outputs] with B_n x B_k blocks, so
 *    bn x bk here is B_k x B_n there, the order Table 4 prints ("BK x BN"); Table 2 uses 32x32,
 *    64x32, 16x32 and 16x16, and a square b x b block is bn = bk = b. A nonzero mask byte keeps the block; a
 *    zero byte removes it, and a removed weight is exactly zero whatever W holds there
 *    (the pruned value is never multiplied, so NaN or Inf in a pruned block has no effect).
 *
 *  - The block-sparse matmul whose cost Sec. 3.3 models (Eq. for P: one unit of work per
 *    surviving block): here written in the PyTorch Linear convention
 *      y[m][n] = sum_k x[m][k] * W~[n][k] + bias[n]
 *    with W stored [out=n][in=k]. The sum runs over k in ascending order in double.
 *
 *  - GELU after fc1 (the DeiT MLP activation; the paper does not state its form, the exact
 *    erf form is used): gelu(y) = y * Phi(y) = 0.5 * y * (1 + erf(y / sqrt(2))), evaluated as
 *    0.5 * y * erfc(-y / sqrt(2)) (the same function; 1 + erf cancels where erf is near -1, erfc
 *    keeps the relative accuracy there).
 *
 *  - Block-sparse packing of the surviving blocks (BSR), Sec. 1 and Sec. 3.3 (only the
 *    surviving blocks are stored and moved): for each row panel r (bn consecutive output
 *    rows), cnt[r] = number of kept blocks, row_ptr = exclusive prefix sum of cnt,
 *    col_idx lists the kept block columns of panel r in ascending order, and blocks[t]
 *    is the bn x bk tile of W copied row-major with its bf16 bits unchanged.
 *
 *  - Round-to-nearest-even conversion of a double to bfloat16 (8 significant bits,
 *    the float32 exponent range, subnormals below 2^-126), written from that definition.
 *
 *  - Block mask from first-order Taylor scores, Sec. 3.1 ("Block-structured Pruning within
 *    layer"): the neuron score S = |W . grad_W f| element by element, a 2D average pooling
 *    with the block as window and stride gives one score per block, the blocks are ranked by
 *    that score and the bottom ones are eliminated at the layer's pruning ratio alpha.
 *    Readings where the paper is silent: the number eliminated is round(alpha * blocks),
 *    half away from zero; equal scores rank by linear block index r * (k/bk) + j, the lower
 *    index first (kept first). The score is the plain average of the definition: each product
 *    |w * g| of a bf16 weight and a float32 gradient is exact in double (8 + 24 significant
 *    bits), the magnitudes are added in row-major order in double and the sum is divided by
 *    bn * bk (relative rounding error below bn * bk * 2^-53).
 *
 * Inputs X and W arrive as bfloat16 bit patterns (the same bits the GPU reads); bias as
 * float32. Widening bf16 -> double is exact.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* bf16 bits -> double: a bf16 value is the upper half of a float32. */
double lpvit_oracle_bf16_to_f64(uint16_t bits) {
  uint32_t u = (uint32_t)bits << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return (double)f;
}

/* double -> bf16 bits, round to nearest, ties to even, from the definition of the format:
 * a finite nonzero bf16 is s * q * 2^(e-7) with integer 128 <= q < 256 (normal) or
 * q < 128 with e = -126 (subnormal); we scale |y| so that the last kept bit has weight 1,
 * round the scaled value to an integer with ties to even, and rescale. */
uint16_t lpvit_oracle_round_bf16(double y) {
  if (isnan(y)) return (uint16_t)0x7FC0;
  const uint16_t sign = signbit(y) ? (uint16_t)0x8000 : (uint16_t)0;
  double a = fabs(y);
  if (isinf(a)) return (uint16_t)(sign | 0x7F80);
  if (a == 0.0) return sign;
  int e;
  (void)frexp(a, &e);          /* a = f * 2^e with 0.5 <= f < 1, so floor(log2 a) = e - 1 */
  int lsb_exp = (e - 1) - 7;   /* weight of the last of 8 significant bits */
  if (lsb_exp < -133) lsb_exp = -133; /* subnormal spacing of bf16 is 2^-133 */
  double q = ldexp(a, -lsb_exp);      /* exact: scaling by a power of two */
  double qi = floor(q);
  double frac = q - qi;
  if (frac > 0.5 || (frac == 0.5 && fmod(qi, 2.0) != 0.0)) qi += 1.0;
  double r = ldexp(qi, lsb_exp);      /* exact */
  if (r > 3.3895313892515355e38) return (uint16_t)(sign | 0x7F80); /* above bf16 max -> inf */
  float rf = (float)r;                /* exact: r has <= 8 significant bits */
  uint32_t u;
  memcpy(&u, &rf, sizeof u);
  return (uint16_t)(sign | (uint16_t)((u >> 16) & 0x7FFF));
}

double lpvit_oracle_gelu(double y) { return 0.5 * y * erfc(-y / sqrt(2.0)); }

/* BSR pack by the definition above, bn x bk blocks. col_idx and blocks must hold
 * (n/bn)*(k/bk) entries. Returns nnzb, or -1 on bad arguments. */
int64_t lpvit_oracle_pack(const uint16_t *W, const uint8_t *mask, int32_t n, int32_t k, int32_t bn, int32_t bk,
                          int32_t *row_ptr, int32_t *col_idx, uint16_t *blocks) {
  if (bn <= 0 || bk <= 0 || n % bn != 0 || k % bk != 0) return -1;
  const int32_t np = n / bn, kb = k / bk;
  int64_t t = 0;
  row_ptr[0] = 0;
  for (int32_t r = 0; r < np; ++r) {
    for (int32_t j = 0; j < kb; ++j) {
      if (mask[(int64_t)r * kb + j] == 0) continue;
      col_idx[t] = j;
      for (int32_t c = 0; c < bn; ++c)
        for (int32_t kk = 0; kk < bk; ++kk)
          blocks[(t * bn + c) * bk + kk] = W[(int64_t)(r * bn + c) * k + (int64_t)j * bk + kk];
      ++t;
    }
    row_ptr[r + 1] = (int32_t)t;
  }
  return t;
}

typedef struct {
  const uint16_t *X;
  int64_t m0, m1, ldx;
  const uint16_t *W;
  const uint8_t *mask;
  int32_t n, k, bn, bk;
  const float *bias;
  int gelu;
  double *Y;
  int64_t ldy;
} linear_job;

static void linear_rows(const linear_job *J) {
  const int32_t kb = J->k / J->bk;
  for (int64_t m = J->m0; m < J->m1; ++m) {
    for (int32_t o = 0; o < J->n; ++o) {
      double acc = 0.0;
      for (int32_t i = 0; i < J->k; ++i) {
        /* W~ = W (.) M: a removed weight is zero, its stored bits are not used */
        const int keep = J->mask[(int64_t)(o / J->bn) * kb + i / J->bk] != 0;
        const double w = keep ? lpvit_oracle_bf16_to_f64(J->W[(int64_t)o * J->k + i]) : 0.0;
        acc += lpvit_oracle_bf16_to_f64(J->X[m * J->ldx + i]) * w;
      }
      if (J->bias) acc += (double)J->bias[o];
      if (J->gelu) acc = lpvit_oracle_gelu(acc);
      J->Y[m * J->ldy + o] = acc;
    }
  }
}

static void *linear_thread(void *arg) {
  linear_rows((const linear_job *)arg);
  return NULL;
}

/* Y[m][n] (double) = [gelu](X (W (.) M)^T + bias). X is [m][ldx] bf16 bits, W [n][k] bf16 bits,
 * mask [n/bn][k/bk] bytes, bias float[n] or NULL. Rows are split across nthreads POSIX threads;
 * each output element is computed by exactly one thread in the same order, so the result does
 * not depend on nthreads. Returns 0, or -1 on bad arguments. */
int lpvit_oracle_linear(const uint16_t *X, int64_t m, int64_t ldx, const uint16_t *W, const uint8_t *mask,
                        int32_t n, int32_t k, int32_t bn, int32_t bk, const float *bias, int gelu, double *Y,
                        int64_t ldy, int nthreads) {
  if (bn <= 0 || bk <= 0 || n % bn != 0 || k % bk != 0 || m < 0 || ldx < k || ldy < n) return -1;
  if (nthreads < 1) nthreads = 1;
  if (nthreads > 256) nthreads = 256;
  if ((int64_t)nthreads > m) nthreads = (int)(m > 0 ? m : 1);
  linear_job jobs[256];
  pthread_t th[256];
  for (int t = 0; t < nthreads; ++t) {
    linear_job J = {X, m * t / nthreads, m * (t + 1) / nthreads, ldx, W, mask, n, k, bn, bk, bias, gelu, Y, ldy};
    jobs[t] = J;
  }
  if (nthreads == 1) {
    linear_rows(&jobs[0]);
    return 0;
  }
  int started = 0;
  for (int t = 0; t < nthreads; ++t) {
    if (pthread_create(&th[t], NULL, linear_thread, &jobs[t]) != 0) break;
    ++started;
  }
  for (int t = started; t < nthreads; ++t) linear_rows(&jobs[t]);
  for (int t = 0; t < started; ++t) pthread_join(th[t], NULL);
  return 0;
}

/* Element-wise double -> bf16 bits (round to nearest even). */
void lpvit_oracle_round_bf16_array(const double *y, uint16_t *out, int64_t count) {
  for (int64_t i = 0; i < count; ++i) out[i] = lpvit_oracle_round_bf16(y[i]);
}

/* Sec. 3.1: block score S'[r][j] = the average over the bn x bk block of |W[i][l] * G[i][l]|, in
 * double (see the header). W: bf16 bits [n][k]; G: float32 [n][k]; out: [n/bn][k/bk]. Returns 0, or
 * -1 for a shape that is not a multiple of the block. */
int lpvit_oracle_block_scores(const uint16_t *W, const float *G, int32_t n, int32_t k, int32_t bn, int32_t bk,
                              double *out) {
  if (bn <= 0 || bk <= 0 || n % bn || k % bk) return -1;
  const int32_t np = n / bn, kb = k / bk;
  for (int32_t r = 0; r < np; ++r) {
    for (int32_t j = 0; j < kb; ++j) {
      double sum = 0.0;
      for (int32_t i = 0; i < bn; ++i) {
        for (int32_t l = 0; l < bk; ++l) {
          const int64_t e = (int64_t)(r * bn + i) * k + (int64_t)j * bk + l;
          sum += fabs(lpvit_oracle_bf16_to_f64(W[e]) * (double)G[e]); /* exact product */
        }
      }
      out[(int64_t)r * kb + j] = sum / ((double)bn * (double)bk);
    }
  }
  return 0;
}

typedef struct {
  double score;
  int64_t index;
} scored_block;

/* higher score first; equal scores: lower linear index first */
static int rank_order(const void *pa, const void *pb) {
  const scored_block *a = (const scored_block *)pa, *b = (const scored_block *)pb;
  if (a->score > b->score) return -1;
  if (a->score < b->score) return 1;
  return (a->index > b->index) - (a->index < b->index);
}

/* Number of blocks eliminated at pruning ratio alpha: round(alpha * count), half away from zero. */
int64_t lpvit_oracle_prune_count(double alpha, int64_t count) {
  const double x = alpha * (double)count;
  return (int64_t)floor(x + 0.5);
}

/* Sec. 3.1: rank the blocks by score and eliminate the bottom `prune` of them. scores: [count];
 * mask out: [count], 1 = kept. Returns 0, or -1 for bad arguments. */
int lpvit_oracle_taylor_mask(const double *scores, int64_t count, int64_t prune, uint8_t *mask) {
  if (count < 0 || prune < 0 || prune > count) return -1;
  scored_block *order = (scored_block *)malloc(sizeof(scored_block) * (size_t)(count > 0 ? count : 1));
  if (!order) return -1;
  for (int64_t t = 0; t < count; ++t) {
    order[t].score = scores[t];
    order[t].index = t;
  }
  qsort(order, (size_t)count, sizeof(scored_block), rank_order);
  for (int64_t t = 0; t < count; ++t) mask[order[t].index] = t < count - prune ? 1 : 0;
  free(order);
  return 0;
}
