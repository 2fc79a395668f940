// mlp.cuh -- host interface of the tensor-core two-layer probe (mlp.cu), used by the step entry points.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace switchsd {

constexpr int kMaxMlpSplit = 16;    // CTAs per cluster splitting K
constexpr int kMaxMlpChunks = 8;    // 64-element K chunks staged per CTA: d <= 16 * 8 * 64 = 8192
constexpr int kMaxMlpHidden = 1024; // H1: at most 16 tiles of 64 units

// K split (cluster size) used for hidden size d.
int mlp_split(int d);
// Whether (d, H1) is within the kernel's limits.
bool mlp_shape_ok(int d, int H1);
// Number of 64-unit tiles of the hidden layer: the partial logits per row written to the workspace.
int mlp_tiles_n(int H1);
// zpart [mlp_tiles_n(H1)][B] <- per-tile partial logits (without b2).  Launched with programmatic
// stream serialization.
cudaError_t launch_mlp_tc(const uint16_t *hidden, const uint16_t *W1, const uint16_t *w2, const float *b1, float *zpart,
                          int B, int d, int H1, cudaStream_t stream);

}  // namespace switchsd
