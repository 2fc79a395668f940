// verify.cu -- switchsd_verify: greedy verification and append (§3.3 "Parallel Verification",
// temperature 0 as in the main experiments), and switchsd_verify_sampled: the same at temperature
// T > 0 (App. A) with the speculative-sampling acceptance rule.
//
// One warp per row.  Lanes test 32 draft indices at a time -- greedy: draft[i] differs from the
// target's greedy token; sampled: u[i] * q[i] is not below p[i] (the product rounded to binary32, q = 1
// for a copy draft) -- and the first set bit of the ballot of rejections is the accepted length a.
// Lanes then append draft[0..a) and the target's token at a (greedy: its argmax; sampled: the caller's
// residual or bonus draw) at ctx[L..L+a] and lane 0 publishes L + a + 1.  The work is O(B k) bytes:
// latency-bound by design.
#include "common.cuh"
#include "index.cuh"

namespace switchsd {


constexpr int kVerifyThreads = 256;

struct VerifyArgs {
    const int32_t *draft;
    const int32_t *target;   // greedy: target argmax [B, k+1]; sampled: the residual / bonus draws [B, k+1]
    const float *p, *q, *u;  // sampled only: target and drafter probabilities (q null: 1) and uniforms [B, k]
    const int32_t *draft_len;
    int32_t *ctx;
    int32_t *lens;
    int32_t *out_accept;
    int32_t *status;
    int32_t B, cap, k;
};

template <bool kSampled>
__global__ void __launch_bounds__(kVerifyThreads) verify_kernel(const VerifyArgs a) {
    const int lane = threadIdx.x & 31;
    const int b = (blockIdx.x * kVerifyThreads + threadIdx.x) >> 5;
    pdl_wait();
    pdl_trigger();
    if (b >= a.B) return;
    const int32_t len = a.draft_len[b];
    const int32_t L = a.lens[b];
    if (len < 0 || len > a.k || L < 1 || L > a.cap) {
        if (lane == 0) {
            a.out_accept[b] = -1;
            if (a.status) a.status[b] = SWITCHSD_ROW_BAD_LEN;
        }
        return;
    }
    const int32_t *dr = a.draft + size_t(b) * a.k;
    const int32_t *tg = a.target + size_t(b) * (a.k + 1);
    int32_t acc = len;
    for (int base = 0; base < len; base += kWarp) {
        const int i = base + lane;
        bool mismatch = false;
        if (i < len) {
            if constexpr (kSampled) {
                const size_t o = size_t(b) * a.k + i;
                const float q = a.q ? a.q[o] : 1.f;
                mismatch = !(__fmul_rn(a.u[o], q) < a.p[o]);
            } else {
                mismatch = dr[i] != tg[i];
            }
        }
        const unsigned m = __ballot_sync(kFull, mismatch);
        if (m) {
            acc = base + __ffs(m) - 1;
            break;
        }
    }
    if (L + acc + 1 > a.cap) {
        if (lane == 0) {
            a.out_accept[b] = -1;
            if (a.status) a.status[b] = SWITCHSD_ROW_CAPACITY;
        }
        return;
    }
    int32_t *row = a.ctx + size_t(b) * size_t(a.cap) + L;
    for (int i = lane; i <= acc; i += kWarp) row[i] = i < acc ? dr[i] : tg[acc];
    if (lane == 0) {
        a.lens[b] = L + acc + 1;
        a.out_accept[b] = acc;
        if (a.status) a.status[b] = SWITCHSD_ROW_OK;
    }
}

}  // namespace switchsd

using namespace switchsd;

extern "C" int switchsd_verify(const int32_t *draft, const int32_t *target_argmax, int32_t *out_accept,
                               const switchsd_verify_params *vp) {
    if (!vp || !draft || !target_argmax || !out_accept || !vp->draft_len || !vp->ctx_tokens || !vp->ctx_lens)
        return SWITCHSD_ERR_ARG;
    if (vp->B < 1 || vp->cap < 4 || (vp->cap & 3) != 0 || vp->k < 1 || vp->k > SWITCHSD_KMAX)
        return SWITCHSD_ERR_SHAPE;
    if (vp->index != nullptr) {
        // verification with insertion of the appended positions into the index (no step)
        return index_launch(vp->index, vp->ctx_tokens, vp->ctx_lens, nullptr, nullptr, nullptr, nullptr, nullptr, 0,
                            0, 0, 0.f, draft,
                            target_argmax, vp->draft_len, out_accept, nullptr, nullptr, nullptr, nullptr, nullptr,
                            nullptr, vp->status, vp->B, vp->cap, 8, vp->k, index_n_min(vp->index),
                            index_n_max(vp->index), 0, 0.f, false, static_cast<cudaStream_t>(vp->stream));
    }
    VerifyArgs a;
    a.draft = draft;
    a.target = target_argmax;
    a.p = a.q = a.u = nullptr;
    a.draft_len = vp->draft_len;
    a.ctx = vp->ctx_tokens;
    a.lens = vp->ctx_lens;
    a.out_accept = out_accept;
    a.status = vp->status;
    a.B = vp->B;
    a.cap = vp->cap;
    a.k = vp->k;
    const int warps_per_block = kVerifyThreads / kWarp;
    const int blocks = (vp->B + warps_per_block - 1) / warps_per_block;
    const cudaError_t e = launch_pdl(verify_kernel<false>, dim3(blocks), dim3(kVerifyThreads), 0,
                                     static_cast<cudaStream_t>(vp->stream), 0u, a);
    return e == cudaSuccess ? SWITCHSD_OK : SWITCHSD_ERR_CUDA;
}

extern "C" int switchsd_verify_sampled(const int32_t *draft, const float *p_draft, const float *q_draft,
                                       const float *u, const int32_t *resample, int32_t *out_accept,
                                       const switchsd_verify_params *vp) {
    if (!vp || !draft || !p_draft || !u || !resample || !out_accept || !vp->draft_len || !vp->ctx_tokens ||
        !vp->ctx_lens)
        return SWITCHSD_ERR_ARG;
    if (vp->B < 1 || vp->cap < 4 || (vp->cap & 3) != 0 || vp->k < 1 || vp->k > SWITCHSD_KMAX)
        return SWITCHSD_ERR_SHAPE;
    if (vp->index != nullptr) {
        // the same rule in the index kernel, which also inserts the appended positions (no step)
        return index_launch(vp->index, vp->ctx_tokens, vp->ctx_lens, nullptr, nullptr, nullptr, nullptr, nullptr, 0,
                            0, 0, 0.f, draft, resample, vp->draft_len, out_accept, nullptr, nullptr, nullptr, nullptr,
                            nullptr, nullptr, vp->status, vp->B, vp->cap, 8, vp->k, index_n_min(vp->index),
                            index_n_max(vp->index), 0, 0.f, false, static_cast<cudaStream_t>(vp->stream), p_draft,
                            q_draft, u);
    }
    VerifyArgs a;
    a.draft = draft;
    a.target = resample;
    a.p = p_draft;
    a.q = q_draft;
    a.u = u;
    a.draft_len = vp->draft_len;
    a.ctx = vp->ctx_tokens;
    a.lens = vp->ctx_lens;
    a.out_accept = out_accept;
    a.status = vp->status;
    a.B = vp->B;
    a.cap = vp->cap;
    a.k = vp->k;
    const int warps_per_block = kVerifyThreads / kWarp;
    const int blocks = (vp->B + warps_per_block - 1) / warps_per_block;
    const cudaError_t e = launch_pdl(verify_kernel<true>, dim3(blocks), dim3(kVerifyThreads), 0,
                                     static_cast<cudaStream_t>(vp->stream), 0u, a);
    return e == cudaSuccess ? SWITCHSD_OK : SWITCHSD_ERR_CUDA;
}

// ------------------------------------------------------------------------------------------------
// switchsd_verify_candidates: the W copy candidates of a row verified at once (§3.3 "Parallel
// Verification with Block-Triangular Attention": the target checks every candidate in one pass and
// the longest validated continuation is kept).  One warp per row; per candidate a ballot gives its
// accepted length, the longest is kept (the most recent, lowest index, on a tie) and appended with the
// target's token after it.
// ------------------------------------------------------------------------------------------------
namespace switchsd {

struct CandVerifyArgs {
    const int32_t *cand, *cand_len, *ncand, *target;
    int32_t *ctx, *lens, *out_accept, *out_choice, *status;
    int32_t B, cap, W, D;
};

__global__ void __launch_bounds__(kVerifyThreads) verify_candidates_kernel(const CandVerifyArgs a) {
    const int lane = threadIdx.x & 31;
    const int b = (blockIdx.x * kVerifyThreads + threadIdx.x) >> 5;
    pdl_wait();
    pdl_trigger();
    if (b >= a.B) return;
    const int32_t L = a.lens[b];
    const int32_t nc = a.ncand[b];
    bool bad = L < 1 || L > a.cap || nc < 0 || nc > a.W;
    for (int w = 0; w < nc && !bad; ++w) {
        const int32_t len = a.cand_len[size_t(b) * a.W + w];
        bad = len < 0 || len > a.D;
    }
    if (bad) {
        if (lane == 0) {
            a.out_accept[b] = -1;
            a.out_choice[b] = 0;
            if (a.status) a.status[b] = SWITCHSD_ROW_BAD_LEN;
        }
        return;
    }
    int32_t best = -1, best_w = 0;
    for (int w = 0; w < (nc > 0 ? nc : 1); ++w) {  // no candidate: one empty one
        const int32_t len = nc > 0 ? a.cand_len[size_t(b) * a.W + w] : 0;
        const int32_t *c = a.cand + (size_t(b) * a.W + w) * a.D;
        const int32_t *t = a.target + (size_t(b) * a.W + w) * (a.D + 1);
        int32_t acc = len;
        for (int base = 0; base < len; base += kWarp) {
            const int i = base + lane;
            const unsigned m = __ballot_sync(kFull, i < len && c[i] != t[i]);
            if (m) {
                acc = base + __ffs(m) - 1;
                break;
            }
        }
        if (acc > best) {
            best = acc;
            best_w = w;
        }
    }
    if (L + best + 1 > a.cap) {
        if (lane == 0) {
            a.out_accept[b] = -1;
            a.out_choice[b] = best_w;
            if (a.status) a.status[b] = SWITCHSD_ROW_CAPACITY;
        }
        return;
    }
    const int32_t *c = a.cand + (size_t(b) * a.W + best_w) * a.D;
    const int32_t *t = a.target + (size_t(b) * a.W + best_w) * (a.D + 1);
    int32_t *row = a.ctx + size_t(b) * size_t(a.cap) + L;
    for (int i = lane; i <= best; i += kWarp) row[i] = i < best ? c[i] : t[best];
    if (lane == 0) {
        a.lens[b] = L + best + 1;
        a.out_accept[b] = best;
        a.out_choice[b] = best_w;
        if (a.status) a.status[b] = SWITCHSD_ROW_OK;
    }
}

}  // namespace switchsd

extern "C" int switchsd_verify_candidates(const int32_t *cand, const int32_t *target, int32_t *out_accept,
                                          int32_t *out_choice, const switchsd_candidates_verify_params *vp) {
    if (!vp || !cand || !target || !out_accept || !out_choice || !vp->cand_len || !vp->ncand || !vp->ctx_tokens ||
        !vp->ctx_lens)
        return SWITCHSD_ERR_ARG;
    if (vp->B < 1 || vp->cap < 4 || (vp->cap & 3) != 0 || vp->W < 1 || vp->W > SWITCHSD_WMAX || vp->D < 1 ||
        vp->D > SWITCHSD_KMAX)
        return SWITCHSD_ERR_SHAPE;
    if (vp->index != nullptr) {
        // the same rule in the index kernel, which also inserts the appended positions (no step)
        IndexCandidates ic;
        ic.W = vp->W;
        ic.D = vp->D;
        ic.pv_cand_len = vp->cand_len;
        ic.out_choice = out_choice;
        ic.out_cand = ic.out_cand_len = ic.out_ncand = nullptr;
        return index_launch(vp->index, vp->ctx_tokens, vp->ctx_lens, nullptr, nullptr, nullptr, nullptr, nullptr, 0,
                            0, 0, 0.f, cand, target, vp->ncand, out_accept, nullptr, nullptr, nullptr, nullptr,
                            nullptr, nullptr, vp->status, vp->B, vp->cap, 8, vp->D, index_n_min(vp->index),
                            index_n_max(vp->index), 0, 0.f, false, static_cast<cudaStream_t>(vp->stream), nullptr,
                            nullptr, nullptr, 1, &ic);
    }
    CandVerifyArgs a;
    a.cand = cand;
    a.cand_len = vp->cand_len;
    a.ncand = vp->ncand;
    a.target = target;
    a.ctx = vp->ctx_tokens;
    a.lens = vp->ctx_lens;
    a.out_accept = out_accept;
    a.out_choice = out_choice;
    a.status = vp->status;
    a.B = vp->B;
    a.cap = vp->cap;
    a.W = vp->W;
    a.D = vp->D;
    const int warps_per_block = kVerifyThreads / kWarp;
    const int blocks = (vp->B + warps_per_block - 1) / warps_per_block;
    const cudaError_t e = launch_pdl(verify_candidates_kernel, dim3(blocks), dim3(kVerifyThreads), 0,
                                     static_cast<cudaStream_t>(vp->stream), 0u, a);
    return e == cudaSuccess ? SWITCHSD_OK : SWITCHSD_ERR_CUDA;
}
