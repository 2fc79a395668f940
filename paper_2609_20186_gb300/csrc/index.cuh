// index.cuh -- internal interface of the incremental n-gram index (index.cu), used by the step and
// verification entry points.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "switchsd.h"

namespace switchsd {

// Candidate mode of the index kernel (switchsd_step_candidates / switchsd_verify_candidates with an
// index): W candidates of up to D tokens.  When verifying, the kernel's pv_draft / pv_target / pv_len
// are the previous candidates [B][W][D], their targets [B][W][D+1] and counts [B], with pv_cand_len
// [B][W] their lengths; out_choice [B] receives the kept candidate.  When stepping, out_cand /
// out_cand_len / out_ncand receive the new candidates (out_draft / out_len are unused).
struct IndexCandidates {
    int32_t W, D;
    const int32_t *pv_cand_len;
    int32_t *out_choice, *out_cand, *out_cand_len, *out_ncand;
};

// One launch of the index kernel on B rows: the verification of the previous draft (when pv_len is
// not null; greedy, or sampled when pv_p is not null: accept while u * q < p in binary32, q null = 1),
// the inserts of the appended tokens' n-grams and, when stepping, the lookup, probe, switch and copy
// draft.  prefetch: the SWITCHSD_PREFETCH_* bits of switchsd_params (the row's length and tail, and
// the linear probe, are then read before the grid-dependency wait).  Linear probe: z1_part null;
// hidden_rows > 1: hidden is [B, hidden_rows, d] and the probe
// reads row a_b (row 0 when nothing was appended).  Two-layer probe: z1_part = the split-K partial
// sums [mlp_S][B][H1p] of W1 h written by the kernel just before, b1 (may be null) and w2 the second
// layer.  Returns a SWITCHSD_* code.
int index_launch(switchsd_index *idx, int32_t *ctx, int32_t *lens, const uint16_t *hidden, const uint16_t *probe_w,
                 const float *z1_part, const float *b1, const uint16_t *w2, int mlp_S, int H1, int H1p, float b2,
                 const int32_t *pv_draft, const int32_t *pv_target, const int32_t *pv_len, int32_t *out_accept,
                 int32_t *out_draft, int32_t *out_len, int32_t *out_mode, float *out_score, int32_t *out_match_n,
                 int32_t *out_match_end, int32_t *status, int B, int cap, int d, int k, int n_min, int n_max, int kappa,
                 float logit_tau, bool stepping, cudaStream_t stream, const float *pv_p = nullptr,
                 const float *pv_q = nullptr, const float *pv_u = nullptr, int hidden_rows = 1,
                 const IndexCandidates *cand = nullptr, int prefetch = 0, unsigned long long *counters = nullptr);

int index_n_min(const switchsd_index *idx);
int index_n_max(const switchsd_index *idx);

}  // namespace switchsd
