// mlp.cuh -- host interface of the tensor-core two-layer probe (mlp.cu), used by the step entry points.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace switchsd {

constexpr int kMaxMlpSplit = 16;    // CTAs splitting K
constexpr int kMaxMlpChunks = 8;    // 64-element K chunks staged per CTA: d <= 16 * 8 * 64 = 8192
constexpr int kMaxMlpHidden = 1024; // H1: at most 16 tiles of 64 units
constexpr int kMlpStagesBeside = 2; // chunks staged at once when the rescan kernel runs beside it

// K split used for hidden size d: the partial sums per (row, unit).
int mlp_split(int d);
// Whether (d, H1) is within the kernel's limits.
bool mlp_shape_ok(int d, int H1);
// H1 rounded up to the 64-unit tile: the row stride of the partial sums.
int mlp_hidden_padded(int H1);
// part [mlp_split(d)][B][mlp_hidden_padded(H1)] <- split-K partial sums of W1 h (fp32; units >= H1 are
// zero).  Launched with programmatic stream serialization; prefetch: the hidden states and W1 may be
// read (and the MMAs run) before the preceding kernel finishes (the caller's guarantee,
// SWITCHSD_PREFETCH_PROBE), and the next kernel is released at once; the stores wait.  stages:
// operand chunks staged at once per CTA (0 or >= the CTA's chunks: all of them; fewer leave shared memory
// to a kernel that runs beside this one).
cudaError_t launch_mlp_tc(const uint16_t *hidden, const uint16_t *W1, float *part, int B, int d, int H1,
                          bool prefetch, cudaStream_t stream, int stages = 0);

}  // namespace switchsd
