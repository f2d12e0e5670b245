// Launchers of the Taylor block-score and rank kernels (Sec. 3.1), shared by the block-mask entry
// point and the pruning-ratio allocation; defined in lpvit_mask.cu.
#pragma once
#include <cstdint>
#include <cuda_runtime.h>

namespace lpvit {

// scores[r][j] = the average of |W * G| over block (r, j) (bn rows by bk columns): each product
// rounded to float32, each block row summed in float32, the row sums summed in float32, the total
// divided by bn * bk in double; within (bn + bk) 2^-24 of the exact average (sums of non-negative
// terms). W bf16 [n][k], G float32 [n][k], both 16-byte aligned.
cudaError_t launch_block_scores(const uint16_t *W, const float *G, int n, int k, int bn, int bk, double *scores,
                                cudaStream_t s);
// For each of `total` blocks: rank[t] = the number of blocks ranked ahead of it (higher score, or
// equal score and lower index), and mask[t] = 1 if rank[t] < keep; either output may be null.
cudaError_t launch_block_rank(const double *scores, int64_t total, int64_t keep, uint8_t *mask, int32_t *rank,
                              cudaStream_t s);

}  // namespace lpvit
