// step_api.cu -- the step entry points of the C ABI: switchsd_step, switchsd_verify_step,
// switchsd_verify_sampled_step, switchsd_step_candidates, switchsd_verify_candidates_step and
// switchsd_workspace_bytes.  Host-side validation, the choice of the split, the shared-memory tiling of
// each CTA's range, the two-layer probe's kernels and the index's kernel; the step kernel itself is
// in step.cu.
#include <cstdlib>

#include "common.cuh"
#include "index.cuh"
#include "mlp.cuh"
#include "step.cuh"

namespace switchsd {

// ------------------------------------------------------------------------------------------------
// Host side.
// ------------------------------------------------------------------------------------------------
static int sm_count_cached() {
    static int counts[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
    if (counts[dev] == 0) {
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
        counts[dev] = n;
    }
    return counts[dev];
}

static bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// CTAs per row: the largest power of two, at most kMaxSplit, that leaves every CTA at least 4096
// candidate ends and keeps the grid within one wave of four CTAs per SM (the step kernel's register
// limit); 1 at least.  Measured on this GPU, per-CTA ranges of 4K-9K ends in a single wave beat both
// smaller ranges (more CTAs per row to reduce and ship) and a second wave.
static int choose_split(int B, int cap) {
    const int sms = sm_count_cached() > 0 ? sm_count_cached() : 148;
    int c = 1;
    while (c < kMaxSplit && cap / (2 * c) >= 4096 && int64_t(B) * (2 * c) <= 4ll * sms) c *= 2;
    return c;
}

// CTAs per row of the rescan kernel: the largest power of two, at most kMaxSplit, that leaves every CTA
// at least 4096 candidate ends while two launches' grids fit on the GPU at once (seven of its CTAs per
// SM), so the next launch's copies are in flight while this one finishes; 1 at least.  Measured in the
// benchmark's launch graph (256 launches): the 32K-context rows 8 CTAs 4.36 us per launch (4: 4.54,
// 16: 6.59), the 8K rows 2 CTAs 3.06 us (1: 3.41, 4: 3.28), the 128K rows 16 CTAs 5.17 us (8: 8.74),
// the 16K rows with the two-layer probe 2 CTAs 10.15 us per step (1: 15.83, 4: 11.45).
static int choose_rescan_split(int B, int cap) {
    const int sms = sm_count_cached() > 0 ? sm_count_cached() : 148;
    int c = 1;
    while (c < kMaxSplit && cap / (2 * c) >= 4096 && 2 * int64_t(B) * (2 * c) <= int64_t(kRescanMinBlocks) * sms)
        c *= 2;
    return c;
}

// Polls of the rescan kernel's wait for the row's messages: kWaitLimit, or the value of the environment
// variable SWITCHSD_DIAG_MESSAGE_WAIT_POLLS when it is set (read once per process).  A diagnostic of the
// bounded-wait path: with 0 the leader gives up at once, reports SWITCHSD_ROW_TIMEOUT for every row, and
// still waits (bounded, kWaitLimit) for the messages in flight before it exits.
static uint32_t msg_wait_polls() {
    static const uint32_t polls = [] {
        const char *v = std::getenv("SWITCHSD_DIAG_MESSAGE_WAIT_POLLS");
        if (v == nullptr || *v == '\0') return kWaitLimit;
        char *end = nullptr;
        const unsigned long n = std::strtoul(v, &end, 10);
        return (end != nullptr && *end == '\0' && n <= kWaitLimit) ? uint32_t(n) : kWaitLimit;
    }();
    return polls;
}

// Candidate-mode outputs of switchsd_step_candidates.
struct CandSpec {
    int32_t W, D;
    int32_t *cand, *cand_len, *ncand;
    const int32_t *pv_cand_len;  // fused verification of the previous candidates (null: none)
    int32_t *out_choice;
};

// ------------------------------------------------------------------------------------------------
// hidden_rows = k + 1 with the two-layer probe.  The probe's tensor-core kernel runs before the step
// kernel, so the state it reads -- row a_b of each row's [k+1, d] block -- is gathered first, by a
// kernel that takes the accepted length a_b by the verification's own rule (the step kernel then
// verifies again and must agree): greedy, the first draft position whose token differs from the
// target's; sampled, the first whose u * q (binary32) is not below p; a_b = draft_len when none.
// Row 0 when nothing is appended: a bad length (ctx_lens outside [1, cap], or above len_bound when set;
// draft_len outside [0, k]) or an append that does not fit in cap.
// ------------------------------------------------------------------------------------------------
constexpr int kGatherThreads = 256;

struct GatherArgs {
    const uint16_t *hidden;  // [B, k + 1, d]
    uint16_t *out;           // [B, d]
    const int32_t *lens, *pv_draft, *pv_target, *pv_len;
    const float *pv_p, *pv_q, *pv_u;  // sampled verification, else NULL
    int32_t cap, d, k, len_bound;
};

__global__ void __launch_bounds__(kGatherThreads) gather_rows_kernel(const GatherArgs g) {
    __shared__ int32_t s_row;
    const int b = blockIdx.x;
    pdl_wait();  // the verification inputs come from the preceding kernels
    pdl_trigger();
    if (threadIdx.x < kWarp) {
        const int lane = threadIdx.x;
        const int32_t L_old = g.lens[b];
        const bool len_ok = L_old >= 1 && L_old <= (g.len_bound > 0 ? min(g.len_bound, g.cap) : g.cap);
        int32_t acc = -1;
        if (len_ok) {
            const int32_t *dr = g.pv_draft + size_t(b) * g.k;
            const int32_t *tg = g.pv_target + size_t(b) * (g.k + 1);
            const int32_t pv_n = g.pv_len[b];
            if (pv_n >= 0 && pv_n <= g.k) {
                bool rej_lo, rej_hi;
                if (g.pv_p != nullptr) {
                    const size_t o = size_t(b) * g.k;
                    rej_lo = lane < pv_n && !(__fmul_rn(g.pv_u[o + lane], g.pv_q ? g.pv_q[o + lane] : 1.f) <
                                              g.pv_p[o + lane]);
                    rej_hi = lane + 32 < pv_n && !(__fmul_rn(g.pv_u[o + lane + 32],
                                                             g.pv_q ? g.pv_q[o + lane + 32] : 1.f) <
                                                   g.pv_p[o + lane + 32]);
                } else {
                    rej_lo = lane < pv_n && dr[lane] != tg[lane];
                    rej_hi = lane + 32 < pv_n && dr[lane + 32] != tg[lane + 32];
                }
                const unsigned m_lo = __ballot_sync(kFull, rej_lo);
                const unsigned m_hi = __ballot_sync(kFull, rej_hi);
                acc = m_lo ? __ffs(m_lo) - 1 : (m_hi ? 32 + __ffs(m_hi) - 1 : pv_n);
                if (L_old + acc + 1 > g.cap) acc = -1;
            }
        }
        if (lane == 0) s_row = acc > 0 ? acc : 0;
    }
    __syncthreads();
    const uint4 *src = reinterpret_cast<const uint4 *>(g.hidden + (size_t(b) * size_t(g.k + 1) + size_t(s_row)) *
                                                                      size_t(g.d));
    uint4 *dst = reinterpret_cast<uint4 *>(g.out + size_t(b) * size_t(g.d));
    for (int i = threadIdx.x; i < (g.d >> 3); i += kGatherThreads) dst[i] = src[i];
}

// Bytes of the two-layer probe's split-K partial sums in the workspace (the gathered states follow).
static size_t mlp_part_bytes(int B, int d, int H1) {
    const size_t floats = size_t(mlp_split(d)) * size_t(B) * size_t(mlp_hidden_padded(H1));
    return (floats * sizeof(float) + 255) / 256 * 256;
}

// Shared validation and launch of switchsd_step / switchsd_verify_step.
static int step_entry(int32_t *ctx_tokens, int32_t *ctx_lens, const uint16_t *hidden, const uint16_t *probe_w,
                      const switchsd_params *p, const int32_t *pv_draft, const int32_t *pv_target,
                      const int32_t *pv_len, int32_t *out_accept, int32_t *out_draft, int32_t *out_len,
                      int32_t *out_mode, float *out_score, const float *pv_p = nullptr,
                      const float *pv_q = nullptr, const float *pv_u = nullptr, const CandSpec *cs = nullptr) {
    if (!p || !ctx_tokens || !ctx_lens || !hidden || !probe_w || !out_mode || !out_score) return SWITCHSD_ERR_ARG;
    if (cs == nullptr && (!out_draft || !out_len)) return SWITCHSD_ERR_ARG;
    if (cs != nullptr) {
        if (!cs->cand || !cs->cand_len || !cs->ncand) return SWITCHSD_ERR_ARG;
        if (cs->W < 1 || cs->W > kMaxCand || cs->D < 1 || cs->D > SWITCHSD_KMAX) return SWITCHSD_ERR_SHAPE;
    }
    if (!aligned16(ctx_tokens) || !aligned16(hidden) || !aligned16(probe_w)) return SWITCHSD_ERR_ARG;
    if (p->probe_kind != SWITCHSD_PROBE_LINEAR && p->probe_kind != SWITCHSD_PROBE_MLP) return SWITCHSD_ERR_ARG;
    if (p->B < 1 || p->B > 65535 || p->cap < 4 || (p->cap & 3) != 0) return SWITCHSD_ERR_SHAPE;
    if (p->d < 8 || (p->d & 7) != 0) return SWITCHSD_ERR_SHAPE;
    if (p->k < 1 || p->k > SWITCHSD_KMAX) return SWITCHSD_ERR_SHAPE;
    if (p->n_min < 1 || p->n_max > SWITCHSD_NMAX || p->n_min > p->n_max) return SWITCHSD_ERR_SHAPE;
    if (p->split != 0 && p->split != 1 && p->split != 2 && p->split != 4 && p->split != 8 && p->split != 16)
        return SWITCHSD_ERR_SHAPE;
    if ((p->prefetch & ~(SWITCHSD_PREFETCH_CONTEXT | SWITCHSD_PREFETCH_PROBE)) != 0) return SWITCHSD_ERR_ARG;
    if (p->len_bound < 0 || p->len_bound > p->cap) return SWITCHSD_ERR_ARG;
    // hidden_rows: 0 / 1, or k + 1 for the fused greedy / sampled verification of one draft
    if (p->hidden_rows != 0 && p->hidden_rows != 1) {
        if (p->hidden_rows != p->k + 1 || pv_len == nullptr || cs != nullptr) return SWITCHSD_ERR_ARG;
    }
    if (p->probe_kind == SWITCHSD_PROBE_MLP) {
        if (!mlp_shape_ok(p->d, p->probe_hidden)) return SWITCHSD_ERR_SHAPE;
        if (!p->workspace || !aligned16(p->workspace) ||
            p->workspace_bytes < switchsd_workspace_bytes(p))
            return SWITCHSD_ERR_ARG;
    }

    cudaStream_t stream = static_cast<cudaStream_t>(p->stream);
    StepArgs args;
    args.ctx = ctx_tokens;
    args.lens = ctx_lens;
    args.hidden = hidden;
    args.probe_w = probe_w;
    args.z1_part = nullptr;
    args.b1 = nullptr;
    args.w2 = nullptr;
    args.mlp_S = args.H1 = args.H1p = 0;
    args.pv_draft = pv_draft;
    args.pv_target = pv_target;
    args.pv_len = pv_len;
    args.pv_p = pv_p;
    args.pv_q = pv_q;
    args.pv_u = pv_u;
    args.out_accept = out_accept;
    args.B = p->B;
    args.cap = p->cap;
    args.d = p->d;
    // candidate mode: a verified candidate appends up to D + 1 tokens, so the staged look-ahead covers D
    args.k = cs ? (p->k > cs->D ? p->k : cs->D) : p->k;
    args.n_min = p->n_min;
    args.n_max = p->n_max;
    args.kappa = p->kappa;
    args.logit_tau = p->logit_tau;
    args.out_draft = out_draft;
    args.out_len = out_len;
    args.out_mode = out_mode;
    args.out_score = out_score;
    args.out_match_n = p->out_match_n;
    args.out_match_end = p->out_match_end;
    args.status = p->status;
    args.prefetch = p->prefetch;
    args.hidden_rows = p->hidden_rows > 1 ? p->hidden_rows : 1;
    args.len_bound = p->len_bound;
    args.counters = cs == nullptr ? reinterpret_cast<unsigned long long *>(p->counters) : nullptr;
    args.msg_wait_polls = kWaitLimit;
    args.wait_late = 0;

    args.probe_words = 0;
    args.hash_words = 0;
    const int split = p->split > 0 ? p->split : choose_split(p->B, p->cap);
    // Tile: the largest CTA range (the last CTA may also cover a k + 1 token append), in one stage
    // up to kSingleTileMax ends (64 KB; one copy, and few enough bytes that a grid of two or four
    // CTAs per SM stays resident in one wave), else a ring of kTileMax stages, as many as the range
    // needs up to kMaxStages and the shared-memory budget.
    const int64_t range = ((int64_t(p->cap) - 1 + split - 1) / split + 3) / 4 * 4 + args.k + 1;
    // candidate mode: a bit per end of the CTA's range, after the stages
    args.W = cs ? cs->W : 0;
    args.D = cs ? cs->D : 0;
    args.bm_words = cs ? int32_t((range + 31) / 32) : 0;
    args.out_cand = cs ? cs->cand : nullptr;
    args.out_cand_len = cs ? cs->cand_len : nullptr;
    args.out_ncand = cs ? cs->ncand : nullptr;
    args.pv_cand_len = cs ? cs->pv_cand_len : nullptr;
    args.out_choice = cs ? cs->out_choice : nullptr;
    const size_t budget = kStageSmemBudget - size_t(args.bm_words) * sizeof(uint32_t);
    if (range <= kSingleTileMax) {
        args.tile = int32_t((range + 3) / 4 * 4);
        args.stages = 1;
    } else {
        args.tile = kTileMax;
        const int64_t need = (range + kTileMax - 1) / kTileMax;
        const int64_t fit = int64_t(budget / ((kHalo + kTileMax + kFwd) * sizeof(int32_t)));
        args.stages = int32_t(need < fit ? need : fit);
        if (args.stages > kMaxStages) args.stages = kMaxStages;
        if (args.stages < 2) args.stages = 2;
    }

    args.b2 = p->b2;
    // The rescan kernel takes the step without the index -- single draft or W candidates, linear probe or
    // the two-layer probe's finish after its first-layer kernel -- when the row's range fits its shared
    // memory; the step kernel takes the rest.
    const bool mlp_probe = p->probe_kind == SWITCHSD_PROBE_MLP;
    const int rsplit = p->split > 0 ? p->split : choose_rescan_split(p->B, p->cap);
    StepArgs ra = args;
    bool rescan = false;
    if (p->index == nullptr && p->cap <= kRescanCapMax) {
        const int64_t rrange = ((int64_t(p->cap) - 1 + rsplit - 1) / rsplit + 3) / 4 * 4;
        const int nv = p->d >> 3;
        const int vper = (nv + rsplit - 1) / rsplit;
        ra.tile = int32_t(rrange);
        ra.stages = 1;
        ra.probe_words = mlp_probe ? 0 : (vper < kProbeStage ? vper : kProbeStage);
        ra.msg_wait_polls = msg_wait_polls();
        ra.bm_words = 0;  // the rescan kernel sizes its own bitmap from the tile
        if (cs == nullptr) {
            ra.W = ra.D = 0;
            ra.out_cand = ra.out_cand_len = ra.out_ncand = ra.out_choice = nullptr;
            ra.pv_cand_len = nullptr;
        }
        ra.hash_words = 0;
        rescan = rrange <= kRescanTileMax && rescan_smem_bytes(ra, rsplit) <= kRescanSmemBudget;
    }
    bool mlp_early = false;  // the first-layer kernel releases the step kernel at its start
    if (mlp_probe) {
        float *part = static_cast<float *>(p->workspace);
        const uint16_t *probe_in = hidden;
        bool probe_pf = (p->prefetch & SWITCHSD_PREFETCH_PROBE) != 0;
        if (args.hidden_rows > 1) {  // gather row a_b of each row first; the step kernel reads no state
            GatherArgs g;
            g.hidden = hidden;
            g.out = reinterpret_cast<uint16_t *>(static_cast<char *>(p->workspace) +
                                                 mlp_part_bytes(p->B, p->d, p->probe_hidden));
            g.lens = ctx_lens;
            g.pv_draft = pv_draft;
            g.pv_target = pv_target;
            g.pv_len = pv_len;
            g.pv_p = pv_p;
            g.pv_q = pv_q;
            g.pv_u = pv_u;
            g.cap = p->cap;
            g.d = p->d;
            g.k = p->k;
            g.len_bound = p->index != nullptr ? 0 : p->len_bound;  // the index ignores the bound
            if (launch_pdl(gather_rows_kernel, dim3(unsigned(p->B)), dim3(kGatherThreads), 0, stream, 0u, g) !=
                cudaSuccess)
                return SWITCHSD_ERR_CUDA;
            probe_in = g.out;
            probe_pf = false;  // the probe kernel's input was just written by the gather
            args.hidden_rows = 1;
        }
        // Beside the rescan kernel the first layer stages two chunks at a time, so that every CTA of the
        // rescan kernel fits on the GPU while it runs (that kernel verifies and scans meanwhile).
        if (launch_mlp_tc(probe_in, probe_w, part, p->B, p->d, p->probe_hidden, probe_pf, stream,
                          rescan ? kMlpStagesBeside : 0) != cudaSuccess)
            return SWITCHSD_ERR_CUDA;
        args.z1_part = part;
        mlp_early = probe_pf;
        args.b1 = p->b1;
        args.w2 = probe_w + size_t(p->probe_hidden) * size_t(p->d);
        args.mlp_S = mlp_split(p->d);
        args.H1 = p->probe_hidden;
        args.H1p = mlp_hidden_padded(p->probe_hidden);
    }
    if (p->index != nullptr) {
        IndexCandidates ic;
        if (cs != nullptr) {
            ic.W = cs->W;
            ic.D = cs->D;
            ic.pv_cand_len = cs->pv_cand_len;
            ic.out_choice = cs->out_choice;
            ic.out_cand = cs->cand;
            ic.out_cand_len = cs->cand_len;
            ic.out_ncand = cs->ncand;
        }
        return index_launch(p->index, ctx_tokens, ctx_lens, hidden, probe_w, args.z1_part, args.b1, args.w2, args.mlp_S,
                            args.H1, args.H1p, args.b2, pv_draft, pv_target, pv_len, out_accept, out_draft, out_len,
                            out_mode, out_score, p->out_match_n, p->out_match_end, p->status, p->B, p->cap, p->d, p->k,
                            p->n_min, p->n_max, p->kappa, p->logit_tau, true, stream, pv_p, pv_q, pv_u,
                            args.hidden_rows, cs != nullptr ? &ic : nullptr, p->prefetch, args.counters);
    }
    if (rescan) {
        ra.z1_part = args.z1_part;
        ra.b1 = args.b1;
        ra.w2 = args.w2;
        ra.mlp_S = args.mlp_S;
        ra.H1 = args.H1;
        ra.H1p = args.H1p;
        ra.hidden_rows = args.hidden_rows;
        // Without the probe prefetch the first-layer kernel launched just above waits for every earlier
        // kernel before it releases this one, so only its own output, the partial sums, needs this
        // launch's wait.  With it, that kernel releases this one at its start: this launch then reads
        // before its wait only what the caller's prefetch bits cover, and everything else after it.
        ra.wait_late = (args.z1_part != nullptr && !mlp_early) ? 1 : 0;
        if (rescan_choose_hash(ra, rsplit, sm_count_cached() > 0 ? sm_count_cached() : 148) != cudaSuccess)
            return SWITCHSD_ERR_CUDA;
        if (launch_rescan_kernel(ra, rsplit, stream) != cudaSuccess) return SWITCHSD_ERR_CUDA;
        return SWITCHSD_OK;
    }
    const cudaError_t e = launch_step_kernel(args, cs != nullptr, split, stream);
    if (e != cudaSuccess) return SWITCHSD_ERR_CUDA;
    return SWITCHSD_OK;
}

}  // namespace switchsd

using namespace switchsd;

extern "C" size_t switchsd_workspace_bytes(const switchsd_params *p) {
    if (!p || p->probe_kind != SWITCHSD_PROBE_MLP || p->B < 1) return 0;
    const int H1 = p->probe_hidden < 1 ? 1 : p->probe_hidden;
    const int d = p->d < 8 ? 8 : p->d;
    size_t bytes = mlp_part_bytes(p->B, d, H1);
    if (p->hidden_rows > 1) bytes += (size_t(p->B) * size_t(d) * sizeof(uint16_t) + 255) / 256 * 256;
    return bytes;
}

extern "C" int switchsd_step(const int32_t *ctx_tokens, const int32_t *ctx_lens, const uint16_t *hidden,
                             const uint16_t *probe_w, const switchsd_params *p, int32_t *out_draft,
                             int32_t *out_len, int32_t *out_mode, float *out_score) {
    return step_entry(const_cast<int32_t *>(ctx_tokens), const_cast<int32_t *>(ctx_lens), hidden, probe_w, p,
                      nullptr, nullptr, nullptr, nullptr, out_draft, out_len, out_mode, out_score);
}

extern "C" int switchsd_verify_step(const int32_t *draft, const int32_t *target_argmax, const int32_t *draft_len,
                                    int32_t *out_accept, int32_t *ctx_tokens, int32_t *ctx_lens,
                                    const uint16_t *hidden, const uint16_t *probe_w, const switchsd_params *p,
                                    int32_t *out_draft, int32_t *out_len, int32_t *out_mode, float *out_score) {
    if (!draft || !target_argmax || !draft_len || !out_accept) return SWITCHSD_ERR_ARG;
    return step_entry(ctx_tokens, ctx_lens, hidden, probe_w, p, draft, target_argmax, draft_len, out_accept,
                      out_draft, out_len, out_mode, out_score);
}

extern "C" int switchsd_step_candidates(const int32_t *ctx_tokens, const int32_t *ctx_lens, const uint16_t *hidden,
                                        const uint16_t *probe_w, const switchsd_params *p, int32_t W, int32_t D,
                                        int32_t *out_cand, int32_t *out_cand_len, int32_t *out_ncand,
                                        int32_t *out_mode, float *out_score) {
    const CandSpec cs{W, D, out_cand, out_cand_len, out_ncand, nullptr, nullptr};
    return step_entry(const_cast<int32_t *>(ctx_tokens), const_cast<int32_t *>(ctx_lens), hidden, probe_w, p,
                      nullptr, nullptr, nullptr, nullptr, nullptr, nullptr, out_mode, out_score, nullptr, nullptr,
                      nullptr, &cs);
}

extern "C" int switchsd_verify_candidates_step(const int32_t *cand, const int32_t *target, const int32_t *cand_len,
                                               const int32_t *ncand, int32_t *out_accept, int32_t *out_choice,
                                               int32_t *ctx_tokens, int32_t *ctx_lens, const uint16_t *hidden,
                                               const uint16_t *probe_w, const switchsd_params *p, int32_t W,
                                               int32_t D, int32_t *out_cand, int32_t *out_cand_len,
                                               int32_t *out_ncand, int32_t *out_mode, float *out_score) {
    if (!cand || !target || !cand_len || !ncand || !out_accept || !out_choice) return SWITCHSD_ERR_ARG;
    const CandSpec cs{W, D, out_cand, out_cand_len, out_ncand, cand_len, out_choice};
    return step_entry(ctx_tokens, ctx_lens, hidden, probe_w, p, cand, target, ncand, out_accept, nullptr, nullptr,
                      out_mode, out_score, nullptr, nullptr, nullptr, &cs);
}

extern "C" int switchsd_verify_sampled_step(const int32_t *draft, const float *p_draft, const float *q_draft,
                                            const float *u, const int32_t *resample, const int32_t *draft_len,
                                            int32_t *out_accept, int32_t *ctx_tokens, int32_t *ctx_lens,
                                            const uint16_t *hidden, const uint16_t *probe_w,
                                            const switchsd_params *p, int32_t *out_draft, int32_t *out_len,
                                            int32_t *out_mode, float *out_score) {
    if (!draft || !p_draft || !u || !resample || !draft_len || !out_accept) return SWITCHSD_ERR_ARG;
    return step_entry(ctx_tokens, ctx_lens, hidden, probe_w, p, draft, resample, draft_len, out_accept, out_draft,
                      out_len, out_mode, out_score, p_draft, q_draft, u);
}
