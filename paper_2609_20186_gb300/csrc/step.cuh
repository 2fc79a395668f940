// step.cuh -- the step kernel's constants, arguments and launcher (step.cu), shared with the entry
// points (step_api.cu).
#pragma once

#include "common.cuh"

namespace switchsd {

constexpr int kStepThreads = 256;
constexpr int kStepWarps = kStepThreads / kWarp;
constexpr int kTileMax = 8192;        // tile of the ring of stages, for ranges above kSingleTileMax
constexpr int kSingleTileMax = 16384; // a CTA range up to this many ends is staged by one copy
constexpr int kHalo = 32;             // look-back staged before a tile: >= SWITCHSD_NMAX, multiple of 4
constexpr int kFwd = SWITCHSD_KMAX;   // look-ahead staged after a tile: the longest copy draft
constexpr int kMaxStages = 6;          // staged tiles in flight per CTA (bounded by shared memory)
constexpr size_t kStageSmemBudget = 200 * 1024;
constexpr int kMaxSplit = 16;
constexpr unsigned long long kTimeoutBit = 1ull << 62;
constexpr int kMaxCand = SWITCHSD_WMAX; // candidate mode: largest W
constexpr int kProbeStage = 256;      // probe words (8 bf16) of w and of h staged per CTA; the rest is read directly
// The rescan kernel (rescan.cu): four warps, at most 64 registers a thread (eight CTAs' worth of an SM's
// registers), so that the next launch's CTAs are resident while this launch finishes; the grid is sized
// for seven CTAs per SM over two launches (a launch spreads unevenly, up to four CTAs on some SMs).
constexpr int kRescanThreads = 128;
constexpr int kRescanWarps = kRescanThreads / kWarp;
constexpr int kRescanMinBlocks = 7;
constexpr int kRescanLaunchBlocks = 8;  // the launch bound: 65,536 / (8 x 128) = 64 registers a thread
constexpr int kRescanTileMax = 16384;  // largest CTA range of the rescan kernel (one bulk copy)
constexpr size_t kRescanSmemBudget = 100 * 1024;
constexpr int kRescanCapMax = 1 << 25;  // the rescan kernel's match keys hold an end below 2^25

static_assert(kHalo >= SWITCHSD_NMAX && kHalo % 4 == 0, "halo must cover the longest n-gram");
static_assert(kFwd % 4 == 0 && kTileMax % 4 == 0, "stages must stay 16-byte aligned");

struct StepArgs {
    int32_t *ctx;            // read through TMA; written (append) by the leader when verifying
    int32_t *lens;           // read; written when verifying
    const uint16_t *hidden;
    const uint16_t *probe_w;
    const float *z1_part;    // two-layer probe: split-K partial sums of W1 h [mlp_S][B][H1p] (workspace), else null
    const float *b1;         // two-layer probe: first-layer biases [H1] (null = zero) and output weights [H1]
    const uint16_t *w2;
    int32_t mlp_S, H1, H1p;
    float b2;
    const int32_t *pv_draft; // previous draft [B, k] / target [B, k+1] / draft length [B]; null = no verify
    const int32_t *pv_target;
    const int32_t *pv_len;
    const float *pv_p, *pv_q, *pv_u;  // sampled verification (T > 0): null = greedy; pv_target then holds
                                      // the residual / bonus draws and pv_q may be null (copy drafts)
    int32_t *out_accept;
    int32_t B, cap, d, k, n_min, n_max, kappa, tile, stages;
    int32_t prefetch;        // SWITCHSD_PREFETCH_* bits: reads that may precede the grid-dependency wait
    int32_t hidden_rows;     // > 1: hidden is [B, hidden_rows, d] and the probe reads row a_b (verifying)
    int32_t len_bound;       // > 0: every row's length is at most this; the ranges are split on it
    float logit_tau;
    int32_t *out_draft, *out_len, *out_mode;
    float *out_score;
    int32_t *out_match_n, *out_match_end, *status;
    int32_t W, D, bm_words;   // candidate mode: W candidates of up to D tokens; bitmap words per CTA
    int32_t *out_cand, *out_cand_len, *out_ncand;
    const int32_t *pv_cand_len;  // candidate mode, verifying: the previous candidates' lengths [B, W]
                                 // (pv_draft [B, W, D], pv_target [B, W, D+1], pv_len = their count [B])
    int32_t *out_choice;         // ... and the kept candidate [B]
    int32_t probe_words;         // rescan kernel: probe words of w and of h staged per CTA
    int32_t hash_words;          // rescan kernel: words of the pre-wait hash bytes of the old ends (one byte
                                 // an end, a multiple of 4 words), 0 = pass 1 hashes the tokens after the wait
    unsigned long long *counters;  // optional per-mode tallies (switchsd_params.counters), else null
    uint32_t msg_wait_polls;     // rescan kernel: polls of the leader's wait for the messages (kWaitLimit
                                 // normally; see msg_wait_polls() in step_api.cu)
    int32_t wait_late;           // rescan kernel, two-layer probe: the kernel just before is the probe's
                                 // first layer, which releases this launch only after its own wait; the
                                 // grid-dependency wait then guards the partial sums alone
};

__device__ __forceinline__ float dot8_bf16(uint4 w, uint4 h, float acc) {
    acc = fmaf(bf16_lo(w.x), bf16_lo(h.x), acc);
    acc = fmaf(bf16_hi(w.x), bf16_hi(h.x), acc);
    acc = fmaf(bf16_lo(w.y), bf16_lo(h.y), acc);
    acc = fmaf(bf16_hi(w.y), bf16_hi(h.y), acc);
    acc = fmaf(bf16_lo(w.z), bf16_lo(h.z), acc);
    acc = fmaf(bf16_hi(w.z), bf16_hi(h.z), acc);
    acc = fmaf(bf16_lo(w.w), bf16_lo(h.w), acc);
    acc = fmaf(bf16_hi(w.w), bf16_hi(h.w), acc);
    return acc;
}

__device__ __forceinline__ void st_cluster_i32(uint32_t addr, int32_t v) {
    asm volatile("st.shared::cluster.s32 [%0], %1;\n" ::"r"(addr), "r"(v) : "memory");
}

// Launches step_kernel<cand> on grid (split, B) as clusters of `split` CTAs, with the shared memory
// that args.stages / args.tile / args.bm_words call for.
cudaError_t launch_step_kernel(const StepArgs &args, bool cand, int split, cudaStream_t stream);

// The rescan kernel (rescan.cu) on grid (split, B): the linear probe, greedy or sampled verification (or
// none), no candidates, no length bound; args.tile >= the largest CTA range, args.probe_words set.
cudaError_t launch_rescan_kernel(const StepArgs &args, int split, cudaStream_t stream);
size_t rescan_smem_bytes(const StepArgs &args, int split);
// Sets args.hash_words: the pre-wait hash table when the grid has at least one CTA per SM (`sms` SMs) and
// the table's shared memory keeps the launch's resident CTAs per SM at min(kRescanMinBlocks, what they are
// without it), else 0.  args.tile, args.z1_part, args.W and args.pv_p must be set.
cudaError_t rescan_choose_hash(StepArgs &args, int split, int sms);

}  // namespace switchsd
