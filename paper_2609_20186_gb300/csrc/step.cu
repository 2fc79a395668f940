// step.cu -- switchsd_step and switchsd_verify_step: n-gram search, probe, switch and copy-draft gather
// for B rows, optionally preceded by the greedy verification and append of the previous draft.
//
// Paper: §3.3 (kappa-gram gate, recency-ranked copy candidates, Eq. 4 decision rule, parallel
// verification, overall framework), Eq. 3 (linear probe), Fig. 1 (three cases).
//
// Layout of the work.  Row b is handled by one thread-block cluster of C CTAs (grid = C x B).  The
// candidate end positions e in [0, L-1) are split into C contiguous 16-byte-aligned ranges.  Each CTA
// stages its range in shared memory with bulk TMA copies (normally one copy: the host sizes the tile to
// the range); a copy also brings kHalo tokens of look-back (for the backward compare) and kFwd tokens
// of look-ahead (for the copy draft).  The copies are issued as soon as the row length is known,
// before any other dependent load, so the whole context is in flight at once.  A position e is a
// candidate when x[e] equals the current token; the thread then compares backwards against the suffix
// (held in shared memory) to get m(e) = the common suffix length, capped at n_max.  The row's answer is
// the maximum of the packed key (m << 32 | e) over candidates with m >= n_min: the largest m first,
// then the most recent e -- exactly the longest-then-most-recent rule.
//
// Fused verification (switchsd_verify_step).  While the copies fly, every CTA of the row recomputes the
// accepted length a of the previous draft (a warp ballot over draft vs target) and the tokens it
// appends, draft[0..a) then target[a].  The split is taken on the length before the append and the
// last CTA's range stretches to the longest possible append, so the copies never wait for the verify.
// Staged positions at or past the old length are patched with the appended tokens (the leader writes
// them to global memory in the same launch, so a copy may see either version).  The leader publishes
// the new length only after every CTA of the cluster has read the old one (cluster barrier phase 1).
//
// After each tile the CTA reduces its best key and, when it improves, keeps that match's continuation
// (the candidate draft) from the staged tile.  The same CTAs compute the linear probe: CTA r dots its
// 1/C slice of the hidden state with the probe weights in fp32.  Each CTA then ships its key, probe
// partial and candidate draft into the leader CTA's shared memory with asynchronous DSMEM stores that
// complete on the leader's mbarrier, and exits; the leader waits (bounded) for all C messages, reduces
// them in a fixed order, applies the switch and writes the winner's draft.  No global scratch, no
// atomics, no global re-read of the context.
#include "common.cuh"
#include "index.cuh"
#include "mlp.cuh"

namespace switchsd {


constexpr int kStepThreads = 256;
constexpr int kStepWarps = kStepThreads / kWarp;
constexpr int kTileMax = 8192;        // largest staged tile (candidate ends)
constexpr int kHalo = 32;             // look-back staged before a tile: >= SWITCHSD_NMAX, multiple of 4
constexpr int kFwd = SWITCHSD_KMAX;   // look-ahead staged after a tile: the longest copy draft
constexpr int kMaxStages = 6;          // staged tiles in flight per CTA (bounded by shared memory)
constexpr size_t kStageSmemBudget = 200 * 1024;
constexpr int kMaxSplit = 16;
constexpr unsigned long long kTimeoutBit = 1ull << 62;
constexpr int kMaxCand = SWITCHSD_WMAX; // candidate mode: largest W
constexpr int kProbeStage = 256;      // probe words (8 bf16) of w and of h staged per CTA; the rest is read directly

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

// Per-CTA message to the leader: a 16-byte header (key, probe partial) and the candidate draft padded
// to whole 16-byte words.
struct alignas(16) Slot {
    unsigned long long key;
    float z;
    int32_t count;             // candidate mode: candidate ends that follow
    int32_t cand[SWITCHSD_KMAX];  // the candidate draft, or (candidate mode) candidate ends, most recent first
};

// kCand: the candidate mode of switchsd_step_candidates -- besides the longest match, every end whose
// common suffix reaches kappa is marked in a per-CTA bitmap; the CTA ships its kMaxCand most recent
// marks and the leader keeps the W most recent of the row.
template <bool kCand>
__global__ void __launch_bounds__(kStepThreads) step_kernel(const StepArgs a) {
    extern __shared__ __align__(128) int32_t tiles[];  // stages x (kHalo + tile + kFwd)
    __shared__ __align__(8) uint64_t bars[kMaxStages];
    __shared__ __align__(8) uint64_t tail_bar;                 // the old tail's small copy
    __shared__ __align__(8) uint64_t probe_bar;                // this CTA's slices of w and h
    __shared__ __align__(8) uint64_t s_done;                   // leader: completes when every slot landed
    __shared__ int32_t s_suf[SWITCHSD_NMAX];
    __shared__ __align__(16) int32_t s_tail[kHalo + 8];        // x[tail_lo .. L_old), tail_lo = roundown4(L_old - kHalo)
    __shared__ int32_t s_app[SWITCHSD_KMAX + 1];               // tokens appended by the verification
    __shared__ int32_t s_ver[4];                               // accepted, new length, verify status, tail landed
    __shared__ int32_t s_split[4];                             // warp 0's split: old length, e_lo, e_hi, tiles
    __shared__ unsigned long long s_wkey[kStepWarps];
    __shared__ float s_wz[kStepWarps];
    __shared__ __align__(16) int32_t s_mine[SWITCHSD_KMAX];    // continuation of this CTA's best match
    __shared__ __align__(16) uint4 s_probe[2 * kProbeStage];   // linear: w then h slices; two-layer: partial sums
    __shared__ Slot s_slot[kMaxSplit];                         // leader: one message per CTA
    __shared__ int32_t s_out[2];                               // leader: winner rank, draft length
    __shared__ __align__(16) int32_t s_cand[kMaxCand];         // candidate mode: this CTA's / the row's ends
    __shared__ int32_t s_ncand;
    __shared__ int32_t s_choice;                               // candidate verification: the kept candidate
    __shared__ int32_t s_probe_late;                           // early probe: its copies did not land in time

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const uint32_t rank = cluster_ctarank();
    const uint32_t C = cluster_nctarank();
    const int b = blockIdx.y;
    const int stage_ints = kHalo + a.tile + kFwd;
    const bool verifying = a.pv_len != nullptr;
    const int kwords = kCand ? (a.W + 3) >> 2 : (a.k + 3) >> 2;  // 16-byte words of a message's payload
    const uint32_t slot_bytes = 16u * uint32_t(1 + kwords);

    if (tid == 0) {
        for (int s = 0; s < a.stages; ++s) mbar_init(&bars[s], 1);
        mbar_init(&tail_bar, 1);
        mbar_init(&probe_bar, 1);
        s_probe_late = 0;
        if (rank == 0) {
            mbar_init(&s_done, 1);
            mbar_arrive_expect_tx(&s_done, slot_bytes * C);
        }
        fence_mbar_init();
    }
    __syncthreads();  // the barriers are initialised before any other thread arms or waits on one
    // Reads named by a prefetch bit go before the grid-dependency wait: the caller guarantees that
    // the kernel immediately before this one does not write them, and the kernels before that one are
    // complete once it runs (each waits on its own predecessors before it lets this one start).  The
    // L2-coherent load keeps a stale L1 line from an earlier grid out of the length.
    const bool pf_ctx = (a.prefetch & SWITCHSD_PREFETCH_CONTEXT) != 0;
    const bool pf_probe = (a.prefetch & SWITCHSD_PREFETCH_PROBE) != 0;

    // Linear probe: this CTA's slice is words [v0, v1) of 8 bf16; the first kProbeStage of them are
    // staged by two bulk copies (issued by thread 64) and used after the scan.  Two-layer probe: this
    // CTA finishes units [u0, u1) of the row -- the S split-K partial sums of each unit, staged the
    // same way when they fit (m_staged), then b1, ReLU and w2.
    uint4 *s_pw = s_probe, *s_ph = s_probe + kProbeStage;
    const bool mlp = a.z1_part != nullptr;
    int v0 = 0, v1 = 0, u0 = 0, u1 = 0, ucnt4 = 0;
    bool m_staged = false;
    if (!mlp) {
        const int nv = a.d >> 3;
        const int per = (nv + int(C) - 1) / int(C);
        v0 = min(nv, int(rank) * per);
        v1 = min(nv, v0 + per);
    } else {
        const int per = ((a.H1 + int(C) - 1) / int(C) + 3) & ~3;
        u0 = min(a.H1, int(rank) * per);
        u1 = min(a.H1, u0 + per);
        ucnt4 = (u1 - u0 + 3) & ~3;  // units staged per partial (H1p >= u0 + ucnt4: rows are padded to 64)
        m_staged = a.mlp_S * ucnt4 <= 2 * kProbeStage * 4;
    }
    const int v_staged = min(v1 - v0, kProbeStage);
    // gather: the probe reads the row a_b of the target's [B, k+1, d] output, known after the verification
    const bool gather = verifying && a.hidden_rows > 1;
    const uint4 *h4 = reinterpret_cast<const uint4 *>(a.hidden + size_t(b) * size_t(gather ? a.hidden_rows : 1) *
                                                                  size_t(a.d));
    const uint4 *w4 = reinterpret_cast<const uint4 *>(a.probe_w);
    auto issue_probe = [&]() {
        if (!mlp) {
            const uint32_t pb = uint32_t(v_staged) * 16u;
            mbar_expect_tx_relaxed(&probe_bar, 2u * pb);
            if (pb > 0) {
                bulk_g2s(s_pw, w4 + v0, pb, &probe_bar);
                bulk_g2s(s_ph, h4 + v0, pb, &probe_bar);
            }
        } else {
            const uint32_t pb = m_staged ? uint32_t(ucnt4) * 4u : 0u;
            mbar_expect_tx_relaxed(&probe_bar, uint32_t(a.mlp_S) * pb);
            float *dst = reinterpret_cast<float *>(s_probe);
            if (pb > 0)
                for (int s = 0; s < a.mlp_S; ++s)
                    bulk_g2s(dst + s * ucnt4, a.z1_part + (size_t(s) * a.B + size_t(b)) * a.H1p + u0, pb, &probe_bar);
        }
    };
    // The partial sums come from the kernel just before this one: never staged before the wait.
    if (pf_probe && !mlp && !gather && tid == 2 * kWarp) issue_probe();
    if (!pf_ctx) pdl_wait();

    // Warp roles until the suffix is known.  Warp 0 reads the row length and issues the copies at
    // once: first the old tail (for the suffix), then the tiles.  Warp 1 verifies the previous draft.
    // Warps 2.. start the probe copies (unless they went before the wait) and take the length from
    // shared memory after the CTA barrier.  The leader publishes the new length once every CTA has
    // arrived on the cluster barrier, so the two warps that read ctx_lens[b] arrive with release
    // semantics (their read is ordered before the leader's write); the others arrive relaxed (the
    // leader's barrier initialisation is published by its own mbarrier-init fence).
    int32_t *row = a.ctx + size_t(b) * size_t(a.cap);
    int32_t L_old = 0, e_lo = 0, e_hi = 0, ntiles = 0, tail_lo = 0, tail_hi = 0;
    bool len_ok = false;
    auto set_split = [&](int32_t L0) {
        // Split on the old length; the last CTA also covers every end the append can add.
        L_old = L0;
        len_ok = (L_old >= 1 && L_old <= a.cap);
        const int32_t E_split = len_ok ? L_old - 1 : 0;
        const int32_t E_max = len_ok ? (verifying ? min(L_old + a.k + 1, a.cap) : L_old) - 1 : 0;
        int32_t chunk = (E_split + int32_t(C) - 1) / int32_t(C);
        chunk = (chunk + 3) & ~3;
        e_lo = min(E_split, int32_t(rank) * chunk);
        e_hi = rank + 1 == C ? E_max : min(E_split, e_lo + chunk);
        ntiles = (e_hi - e_lo + a.tile - 1) / a.tile;
        tail_lo = max(0, (L_old - kHalo) & ~3);
        tail_hi = len_ok ? (L_old + 3) & ~3 : tail_lo;  // <= cap since cap % 4 == 0
    };
    // Stage tile t: tokens [max(0, t0 - kHalo), min(roundup4(t1 + kFwd), cap)) land so that token p
    // sits at stage[kHalo + p - t0].  cap % 4 == 0 keeps every bound 16-byte aligned.
    auto issue = [&](int t) {
        const int s = t % a.stages;
        const int32_t t0 = e_lo + t * a.tile;
        const int32_t t1 = min(e_hi, t0 + a.tile);
        const int32_t lo = max(0, t0 - kHalo);
        const int32_t hi = min((t1 + kFwd + 3) & ~3, a.cap);
        const uint32_t bytes = uint32_t(hi - lo) * 4u;
        mbar_expect_tx_relaxed(&bars[s], bytes);
        bulk_g2s_hint(tiles + s * stage_ints + (kHalo + lo - t0), row + lo, bytes, &bars[s], l2_evict_first_policy());
    };
    // With a length bound the ranges are split on the bound, so the tile copies leave before the row
    // length is read; the length then gives the tail, the verification and the end of the scan (a row
    // longer than the bound is a bad length).
    const bool bounded = a.len_bound > 0;
    if (warp < 2) {
        if (bounded) {
            set_split(a.len_bound);
            if (warp == 0 && lane == 0)
                for (int t = 0; t < min(ntiles, a.stages); ++t) issue(t);
            L_old = __ldcg(a.lens + b);
            len_ok = L_old >= 1 && L_old <= a.len_bound && L_old <= a.cap;
            tail_lo = max(0, (L_old - kHalo) & ~3);
            tail_hi = len_ok ? (L_old + 3) & ~3 : tail_lo;
        } else {
            set_split(__ldcg(a.lens + b));
        }
    }
    // Every thread arrives now, before issuing anything else: only the length read has to precede
    // the leader's write of the new length.
    if (warp < 2)
        cluster_arrive_release();
    else
        cluster_arrive_relaxed();

    if (warp == 0) {
        if (lane == 0) {
            const uint32_t tb = uint32_t(tail_hi - tail_lo) * 4u;
            mbar_expect_tx_relaxed(&tail_bar, tb);
            if (tb > 0) bulk_g2s_hint(s_tail, row + tail_lo, tb, &tail_bar, l2_evict_first_policy());
            if (!bounded)
                for (int t = 0; t < min(ntiles, a.stages); ++t) issue(t);
            s_split[0] = L_old;
            s_split[1] = e_lo;
            s_split[2] = e_hi;
            s_split[3] = ntiles;
        }
    }
    // A prefetched linear probe is finished before the wait by warps 2.. (idle until then): its slice was
    // copied at the very start and nothing the preceding kernel writes enters it.
    const bool early_probe = pf_probe && !mlp && !gather;
    if (early_probe && warp >= 2) {
        float zp = 0.f;
        const bool in = mbar_wait(&probe_bar, 0);
        if (in)
            for (int i = tid - 2 * kWarp; i < v_staged; i += kStepThreads - 2 * kWarp)
                zp = dot8_bf16(s_pw[i], s_ph[i], zp);
        for (int v = v0 + v_staged + tid - 2 * kWarp; v < v1; v += kStepThreads - 2 * kWarp)
            zp = dot8_bf16(__ldg(w4 + v), __ldg(h4 + v), zp);
        zp = warp_sum_f32(zp);
        if (lane == 0) s_wz[warp] = zp;
        if (!in && lane == 0) s_probe_late = 1;  // benign race: every writer stores 1
    } else if (early_probe && lane == 0) {
        s_wz[warp] = 0.f;  // warps 0 and 1 hold no share of the early probe
    }
    if (pf_ctx) pdl_wait();  // the previous draft and the target (and all that no bit names) come after this
    pdl_trigger();           // the next kernel may start launching
    float m_b1 = 0.f, m_w2 = 0.f;  // two-layer probe: this thread's first unit, loaded while the copies fly
    if (mlp && tid < u1 - u0) {
        m_b1 = a.b1 ? a.b1[u0 + tid] : 0.f;
        m_w2 = bf16_lo(uint32_t(a.w2[u0 + tid]));
    }
    if (warp == 1) {
        // Verification of the previous draft (every CTA of the row computes the same result).  Lane i
        // reads draft[i], draft[i+32], target[i], target[i+32] and (lane 0) target[64].
        int32_t acc = -1, L = L_old, vst = len_ok ? SWITCHSD_ROW_OK : SWITCHSD_ROW_BAD_LEN;
        if (kCand && verifying && len_ok) {
            // The W previous candidates verified at once (§3.3): lane i tests positions i and i + 32
            // of every candidate; the longest accepted one is kept (the lowest index on a tie).  Every
            // slot's tokens are loaded without waiting for its length, so the loads go out together.
            const int32_t nc = a.pv_len[b];
            int32_t best = -1, best_w = 0;
            bool badlen = nc < 0 || nc > a.W;
            const int ncx = badlen ? 0 : (nc > 0 ? nc : 1);
#pragma unroll
            for (int w = 0; w < kMaxCand; ++w) {
                if (w < ncx) {
                    const size_t o = size_t(b) * a.W + w;
                    const int32_t *c = a.pv_draft + o * a.D;
                    const int32_t *t = a.pv_target + o * (a.D + 1);
                    const int32_t c_lo = lane < a.D ? c[lane] : 0, c_hi = lane + 32 < a.D ? c[lane + 32] : 0;
                    const int32_t t_lo = lane < a.D ? t[lane] : 0, t_hi = lane + 32 < a.D ? t[lane + 32] : 0;
                    const int32_t len = nc > 0 ? a.pv_cand_len[o] : 0;
                    badlen |= len < 0 || len > a.D;
                    const unsigned m_lo = __ballot_sync(kFull, lane < len && c_lo != t_lo);
                    const unsigned m_hi = __ballot_sync(kFull, lane + 32 < len && c_hi != t_hi);
                    const int32_t acc_w = m_lo ? __ffs(m_lo) - 1 : (m_hi ? 32 + __ffs(m_hi) - 1 : len);
                    if (acc_w > best) {
                        best = acc_w;
                        best_w = w;
                    }
                }
            }
            if (badlen) {
                vst = SWITCHSD_ROW_BAD_LEN;
            } else if (L_old + best + 1 > a.cap) {
                vst = SWITCHSD_ROW_CAPACITY;
            } else {
                const size_t o = size_t(b) * a.W + best_w;
                const int32_t *c = a.pv_draft + o * a.D;
                if (lane < best) s_app[lane] = c[lane];
                if (lane + 32 < best) s_app[lane + 32] = c[lane + 32];
                if (lane == 0) s_app[best] = a.pv_target[o * (a.D + 1) + best];
                acc = best;
                L = L_old + best + 1;
            }
            if (lane == 0) s_choice = best_w;
        } else if (verifying && len_ok) {
            const int32_t *dr = a.pv_draft + size_t(b) * a.k;
            const int32_t *tg = a.pv_target + size_t(b) * (a.k + 1);
            const int32_t pv_n = a.pv_len[b];
            const int32_t d_lo = lane < a.k ? dr[lane] : 0;
            const int32_t d_hi = lane + 32 < a.k ? dr[lane + 32] : 0;
            const int32_t t_lo = lane <= a.k ? tg[lane] : 0;
            const int32_t t_hi = lane + 32 <= a.k ? tg[lane + 32] : 0;
            const int32_t t_top = (lane == 0 && a.k >= 64) ? tg[64] : 0;
            if (pv_n < 0 || pv_n > a.k) {
                vst = SWITCHSD_ROW_BAD_LEN;
            } else {
                // greedy: a draft token is rejected when it differs from the target's; sampled: when
                // u * q (binary32) is not below p
                bool rej_lo = lane < pv_n && d_lo != t_lo, rej_hi = lane + 32 < pv_n && d_hi != t_hi;
                if (a.pv_p != nullptr) {
                    const size_t o = size_t(b) * a.k;
                    rej_lo = lane < pv_n &&
                             !(__fmul_rn(a.pv_u[o + lane], a.pv_q ? a.pv_q[o + lane] : 1.f) < a.pv_p[o + lane]);
                    rej_hi = lane + 32 < pv_n && !(__fmul_rn(a.pv_u[o + lane + 32],
                                                            a.pv_q ? a.pv_q[o + lane + 32] : 1.f) <
                                                   a.pv_p[o + lane + 32]);
                }
                const unsigned m_lo = __ballot_sync(kFull, rej_lo);
                const unsigned m_hi = __ballot_sync(kFull, rej_hi);
                acc = m_lo ? __ffs(m_lo) - 1 : (m_hi ? 32 + __ffs(m_hi) - 1 : pv_n);
                if (L_old + acc + 1 > a.cap) {
                    vst = SWITCHSD_ROW_CAPACITY;
                    acc = -1;
                } else {
                    // s_app[i] = draft[i] for i < acc, target[acc] at i = acc
                    const int32_t t_acc =
                        __shfl_sync(kFull, acc < 32 ? t_lo : (acc < 64 ? t_hi : t_top), acc & 31);
                    if (lane < acc) s_app[lane] = d_lo;
                    if (lane + 32 < acc) s_app[lane + 32] = d_hi;
                    if (lane == 0) s_app[acc] = t_acc;
                    L = L_old + acc + 1;
                }
            }
        }
        if (lane == 0) {
            s_ver[0] = acc;
            s_ver[1] = L;
            s_ver[2] = vst;
            if (gather) {  // the probe's slice of hidden row a_b (row 0 when nothing was appended)
                h4 += size_t(acc > 0 ? acc : 0) * size_t(a.d >> 3);
                issue_probe();
            }
        }
    } else if (warp >= 2) {
        if ((!pf_probe || mlp) && !gather && tid == 2 * kWarp) issue_probe();
        if (kCand) {
            uint32_t *bm = reinterpret_cast<uint32_t *>(tiles + a.stages * stage_ints);
            for (int i = tid - 2 * kWarp; i < a.bm_words; i += kStepThreads - 2 * kWarp) bm[i] = 0u;
        }
    }
    // Warps 0 and 1 meet (named barrier 1, 64 threads): the suffix needs the old tail and the append.
    if (warp < 2) {
        asm volatile("bar.sync 1, 64;\n" ::: "memory");
        if (warp == 0) {
            const bool tail_in = tail_hi == tail_lo || mbar_wait(&tail_bar, 0);
            const int32_t L = s_ver[1];
            const int32_t p = L - 1 - lane;  // suffix position; p >= L_old - kHalo since L >= L_old
            int32_t v = 0;
            if (p >= L_old)
                v = s_app[p - L_old];
            else if (len_ok && p >= 0 && tail_in)
                v = s_tail[p - tail_lo];
            s_suf[lane] = v;
            if (lane == 0) s_ver[3] = tail_in;
        }
    }
    __syncthreads();  // suffix, verification and old length visible
    if (warp >= 2) {
        L_old = s_split[0];
        e_lo = s_split[1];
        e_hi = s_split[2];
        ntiles = s_split[3];
        len_ok = (L_old >= 1 && L_old <= (a.len_bound > 0 ? min(a.len_bound, a.cap) : a.cap));
        tail_lo = max(0, (L_old - kHalo) & ~3);
        tail_hi = len_ok ? (L_old + 3) & ~3 : tail_lo;
    }

    const int32_t acc = s_ver[0], L = s_ver[1];
    const int32_t E = len_ok ? L - 1 : 0;  // candidate ends after the append: [0, E)
    if (gather && !(warp == 1 && lane == 0)) h4 += size_t(acc > 0 ? acc : 0) * size_t(a.d >> 3);
    const int32_t s0 = s_suf[0], s1 = s_suf[1];
    const int32_t n_max = a.n_max, n_min = a.n_min;
    // With n_min >= 2 a candidate must match the last two tokens, so the filter tests both (exact:
    // the back-compare then starts at m = 2).  m0 is the length the filter has already checked.
    const bool pair = n_min >= 2;
    const int32_t m0 = pair ? 2 : 1;
    const int32_t kappa_c = a.kappa > 0 ? a.kappa : n_min;  // candidate mode: the gate length
    unsigned long long best = 0;  // CTA-uniform; real keys have m >= n_min >= 1, so 0 = no match
    bool bad = s_ver[3] == 0;     // CTA-uniform: a copy did not land in time
    for (int t = 0; t < ntiles && !bad; ++t) {
        const int s = t % a.stages;
        const bool landed = mbar_wait(&bars[s], uint32_t(t / a.stages) & 1u);
        const int32_t t0 = e_lo + t * a.tile;
        const int32_t tile_end = min(e_hi, t0 + a.tile);
        const int32_t t1 = min(tile_end, E);  // ends scanned in this tile
        int32_t *stage = tiles + s * stage_ints;
        const int32_t off = kHalo - t0;  // stage[off + p] = x[p] over the staged range
        if (verifying) {
            const int32_t lo = max(0, t0 - kHalo), hi = min((tile_end + kFwd + 3) & ~3, a.cap);
            const int32_t p0 = max(lo, L_old), p1 = min(hi, L);
            if (p0 < p1) {  // CTA-uniform
                if (landed)
                    for (int32_t p = p0 + tid; p < p1; p += kStepThreads) stage[off + p] = s_app[p - L_old];
                __syncthreads();
            }
        }
        unsigned long long mine = 0;
        if (landed) {
            const int32_t n4 = (t1 - t0 + 3) >> 2;
            const int4 *g4 = reinterpret_cast<const int4 *>(stage + kHalo);
            // The bound is warp-uniform (g0 - lane is the warp's first word); lanes past the end read
            // zeros and their ends fail e < t1.
            for (int32_t g0 = tid; g0 - lane < n4; g0 += 4 * kStepThreads) {
                int4 v[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int32_t g = g0 + u * kStepThreads;
                    v[u] = g < n4 ? g4[g] : make_int4(0, 0, 0, 0);
                }
                // One predicate for the four words first: most words hold no first-token hit, and the
                // bit masks are only built for those that do.
                bool any = false;
#pragma unroll
                for (int u = 0; u < 4; ++u)
                    any |= (v[u].x == s0) | (v[u].y == s0) | (v[u].z == s0) | (v[u].w == s0);
                if (!any) continue;
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int32_t g = g0 + u * kStepThreads;
                    const int32_t e4 = t0 + 4 * g;
                    unsigned hits = unsigned(v[u].x == s0) | (unsigned(v[u].y == s0) << 1) |
                                    (unsigned(v[u].z == s0) << 2) | (unsigned(v[u].w == s0) << 3);
                    if (pair && hits != 0u) {
                        // x[e - 1] sits in this word for three of the four ends; for the first it is
                        // the staged token before the word (unset at e4 = 0, where no 2-gram ends).
                        unsigned pm = (unsigned(v[u].x == s1) << 1) | (unsigned(v[u].y == s1) << 2) |
                                      (unsigned(v[u].z == s1) << 3);
                        if ((hits & 1u) != 0u && g < n4) pm |= unsigned(stage[kHalo + 4 * g - 1] == s1);
                        hits &= pm;
                    }
                    while (hits) {
                        const int32_t e = e4 + __ffs(hits) - 1;
                        hits &= hits - 1;
                        if (e >= t1) break;
                        const int32_t lim = min(n_max, e + 1);
                        if (lim < m0) continue;
                        int32_t m = m0;
                        while (m < lim && stage[off + e - m] == s_suf[m]) ++m;
                        if (m >= n_min) {
                            const unsigned long long key =
                                (static_cast<unsigned long long>(m) << 32) | uint32_t(e);
                            mine = key > mine ? key : mine;
                        }
                        if (kCand && m >= kappa_c) {
                            uint32_t *bm = reinterpret_cast<uint32_t *>(tiles + a.stages * stage_ints);
                            atomicOr(&bm[(e - e_lo) >> 5], 1u << ((e - e_lo) & 31));
                        }
                    }
                }
            }
        }
        // Tile reduction; on improvement the threads that will ship the candidate copy it while the
        // tile is still staged (thread j owns candidate words j-1).
        mine = warp_max_u64(mine);
        if (lane == 0) s_wkey[warp] = mine;
        bad = __syncthreads_or(!landed);
        unsigned long long tile_best = 0;
#pragma unroll
        for (int w = 0; w < kStepWarps; ++w) tile_best = s_wkey[w] > tile_best ? s_wkey[w] : tile_best;
        if (!bad && tile_best > best) {
            best = tile_best;
            if (!kCand && tid >= 1 && tid <= kwords) {
                const int32_t e = int32_t(best & 0xffffffffu);
                const int32_t len = min(a.k, L - 1 - e);
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const int i = 4 * (tid - 1) + q;
                    s_mine[i] = i < len ? stage[off + e + 1 + i] : 0;
                }
            }
        }
        if (!bad && t + a.stages < ntiles) {
            __syncthreads();  // stage s and s_wkey are free again
            if (tid == 0) {
                asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
                issue(t + a.stages);
            }
        }
    }
    if (bad) {
        best = kTimeoutBit;
        // Give the copies still in flight a second bounded wait before the CTA's memory goes away.
        if (tid == 0) {
            for (int u = 0; u < min(ntiles, a.stages); ++u) (void)mbar_wait(&bars[u], 0u);
            (void)mbar_wait(&tail_bar, 0u);
        }
    }

    // The probe slice (staged during the scan) unless it was finished before the wait, then the CTA's
    // partial in a fixed order.
    float zp = 0.f;
    const bool probe_in = early_probe ? s_probe_late == 0 : mbar_wait(&probe_bar, 0);
    if (early_probe) {
    } else if (!mlp) {
        if (probe_in)
            for (int i = tid; i < v_staged; i += kStepThreads) zp = dot8_bf16(s_pw[i], s_ph[i], zp);
        for (int v = v0 + v_staged + tid; v < v1; v += kStepThreads)
            zp = dot8_bf16(__ldg(w4 + v), __ldg(h4 + v), zp);
    } else {
        const float *sp = reinterpret_cast<const float *>(s_probe);
        for (int j = tid; j < u1 - u0; j += kStepThreads) {
            float z1 = 0.f;  // the S partial sums in order
            if (m_staged) {
                for (int s = 0; s < a.mlp_S; ++s) z1 += sp[s * ucnt4 + j];
            } else {
                for (int s = 0; s < a.mlp_S; ++s) z1 += a.z1_part[(size_t(s) * a.B + size_t(b)) * a.H1p + u0 + j];
            }
            const float bias = j < kStepThreads ? m_b1 : (a.b1 ? a.b1[u0 + j] : 0.f);
            const float w2 = j < kStepThreads ? m_w2 : bf16_lo(uint32_t(a.w2[u0 + j]));
            zp = fmaf(w2, fmaxf(z1 + bias, 0.f), zp);
        }
    }
    if (!probe_in && tid == 0) {
        best = kTimeoutBit;
        (void)mbar_wait(&probe_bar, 0);  // a second bounded wait before the CTA's memory goes away
    }
    if (!early_probe) {
        zp = warp_sum_f32(zp);
        if (lane == 0) s_wz[warp] = zp;
    }
    if (kCand && warp == 0) {
        // The CTA's most recent marked ends: 32 bitmap words per pass from the top; lane i holds word
        // top - i, and a prefix sum of the popcounts ranks its bits after those of higher words.
        const uint32_t *bm = reinterpret_cast<const uint32_t *>(tiles + a.stages * stage_ints);
        int found = 0;
        for (int top = a.bm_words - 1; top >= 0 && found < a.W; top -= kWarp) {
            const int idx = top - lane;
            const uint32_t wd = (idx >= 0 && !bad) ? bm[idx] : 0u;
            const int c = __popc(wd);
            int incl = c;
#pragma unroll
            for (int o = 1; o < kWarp; o <<= 1) {
                const int t = __shfl_up_sync(kFull, incl, o);
                if (lane >= o) incl += t;
            }
            int r = found + incl - c;
            uint32_t w2 = wd;
            while (w2 != 0u && r < a.W) {
                const int bit = 31 - __clz(w2);
                w2 &= ~(1u << bit);
                s_cand[r++] = e_lo + idx * 32 + bit;
            }
            found += __shfl_sync(kFull, incl, kWarp - 1);
        }
        if (lane == 0) s_ncand = found < a.W ? found : a.W;
    }
    __syncthreads();
    float cta_z = 0.f;
    if (warp == 0) cta_z = warp_sum_f32(lane < kStepWarps ? s_wz[lane] : 0.f);

    // Every CTA has started and read ctx_lens[b] once this returns (they all arrived long ago).
    cluster_wait_acquire();
    if (rank == 0 && verifying) {
        // The leader publishes the append; the other CTAs only patched their staged copies.
        for (int i = tid; i <= acc; i += kStepThreads) row[L_old + i] = s_app[i];
        if (tid == 0 && len_ok) {
            a.lens[b] = L;
            a.out_accept[b] = acc;
        }
    }

    // Ship this CTA's message to the leader: asynchronous DSMEM stores that complete on its barrier.
    const uint32_t done_addr = map_to_rank(&s_done, 0);
    if (tid == 0) {
        uint4 h;
        h.x = uint32_t(best & 0xffffffffu);
        h.y = uint32_t(best >> 32);
        h.z = __float_as_uint(cta_z);
        h.w = kCand ? uint32_t(s_ncand) : 0u;
        st_async_v4(map_to_rank(&s_slot[rank], 0), h, done_addr);
    } else if (tid <= kwords) {
        const uint4 v = kCand ? *reinterpret_cast<const uint4 *>(&s_cand[4 * (tid - 1)])
                              : *reinterpret_cast<const uint4 *>(&s_mine[4 * (tid - 1)]);
        st_async_v4(map_to_rank(&s_slot[rank].cand[4 * (tid - 1)], 0), v, done_addr);
    }
    if (rank != 0) return;

    if (warp == 0) {
        // Bounded wait for every CTA's message (C x slot_bytes of transaction); lane r reads CTA r's.
        // The largest key wins (CTAs tie only at 0, no match: their ends differ), and the probe
        // partials are summed by a fixed shuffle tree, so the result is the same on every run.
        const bool all_in = __all_sync(kFull, mbar_wait(&s_done, 0));
        unsigned long long k_r = 0ull;
        float z_r = 0.f;
        if (all_in && uint32_t(lane) < C) {
            k_r = s_slot[lane].key;
            z_r = s_slot[lane].z;
        }
        const unsigned long long key = all_in ? warp_max_u64(k_r) : kTimeoutBit;
        const unsigned at = __ballot_sync(kFull, uint32_t(lane) < C && k_r == key);
        const uint32_t win = at != 0u ? uint32_t(__ffs(at) - 1) : 0u;
        float z = warp_sum_f32(z_r);
        if (mlp) z += a.b2;
        const bool timeout = (key & kTimeoutBit) != 0;
        const bool hit = len_ok && !timeout && key != 0;
        const int32_t n = hit ? int32_t(key >> 32) : 0;
        const int32_t e = hit ? int32_t(key & 0xffffffffu) : -1;
        const int32_t kappa = a.kappa > 0 ? a.kappa : a.n_min;
        int32_t ncand = 0;  // candidate mode: the row's candidates, merged from the most recent CTA down
        if (kCand) {
            if (lane == 0 && hit) {
                for (int r = int(C) - 1; r >= 0 && ncand < a.W; --r) {
                    const int c = s_slot[r].count;
                    for (int i = 0; i < c && ncand < a.W; ++i) s_cand[ncand++] = s_slot[r].cand[i];
                }
            }
            ncand = __shfl_sync(kFull, ncand, 0);
        }
        const bool gate = kCand ? ncand > 0 : n >= kappa;
        int32_t mode = SWITCHSD_MODE_NO_REP;
        if (hit) mode = (gate && z >= a.logit_tau) ? SWITCHSD_MODE_COPY : SWITCHSD_MODE_REP_NO_COPY;
        const int32_t len = (!kCand && mode == SWITCHSD_MODE_COPY) ? min(a.k, L - 1 - e) : 0;
        if (lane == 0) {
            s_out[0] = int32_t(win);
            s_out[1] = len;
            if (kCand) s_ncand = mode == SWITCHSD_MODE_COPY ? ncand : 0;
            a.out_mode[b] = mode;
            if (!kCand) a.out_len[b] = len;
            a.out_score[b] = z;
            if (a.out_match_n) a.out_match_n[b] = n;
            if (a.out_match_end) a.out_match_end[b] = e;
            if (verifying && !len_ok) a.out_accept[b] = -1;
            if (kCand && verifying && a.out_choice) a.out_choice[b] = len_ok ? s_choice : 0;
            if (a.status) {
                int32_t st = s_ver[2];
                if (st == SWITCHSD_ROW_OK && timeout) st = SWITCHSD_ROW_TIMEOUT;
                a.status[b] = st;
            }
        }
        // The copy draft from the winner's message (every lane knows win and len).
        if (!kCand)
            for (int i = lane; i < len; i += kWarp) a.out_draft[size_t(b) * a.k + i] = s_slot[win].cand[i];
    }
    if (kCand) {
        __syncthreads();
        // The candidates' continuations, read from the row (the leader's append, if any, is visible
        // to its threads after the barrier).
        const int nc = s_ncand;
        if (tid == 0) a.out_ncand[b] = nc;
        for (int t = tid; t < nc * a.D; t += kStepThreads) {
            const int w = t / a.D, i = t - w * a.D;
            const int32_t ew = s_cand[w];
            const int32_t lw = min(a.D, L - 1 - ew);
            if (i == 0) a.out_cand_len[size_t(b) * a.W + w] = lw;
            if (i < lw) a.out_cand[(size_t(b) * a.W + w) * a.D + i] = row[ew + 1 + i];
        }
    }
}

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

// CTAs per row: the smallest power of two giving at least two CTAs per SM over the batch, with at
// least 1024 tokens of capacity per CTA, at most kMaxSplit.
static int choose_split(int B, int cap) {
    const int sms = sm_count_cached() > 0 ? sm_count_cached() : 148;
    int c = 1;
    while (c < kMaxSplit && int64_t(B) * c < 2ll * sms && cap / (2 * c) >= 1024) c *= 2;
    return c;
}

template <bool kCand>
static cudaError_t launch_step(const StepArgs &args, int split, cudaStream_t stream) {
    static bool attr_done[64] = {false};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && !attr_done[dev]) {
        cudaError_t e = cudaFuncSetAttribute(step_kernel<kCand>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        if (e != cudaSuccess) return e;
        e = cudaFuncSetAttribute(step_kernel<kCand>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 int(kStageSmemBudget));
        if (e != cudaSuccess) return e;
        attr_done[dev] = true;
    }
    const size_t smem = size_t(args.stages) * (kHalo + args.tile + kFwd) * sizeof(int32_t) +
                        (kCand ? size_t(args.bm_words) * sizeof(uint32_t) : 0);
    return launch_pdl(step_kernel<kCand>, dim3(unsigned(split), unsigned(args.B), 1), dim3(kStepThreads, 1, 1),
                      smem, stream, unsigned(split), args);
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

    const int split = p->split > 0 ? p->split : choose_split(p->B, p->cap);
    // Tile: the largest CTA range (the last CTA may also cover a k + 1 token append), in one stage
    // when it fits, else a ring of kTileMax stages, as many as the range needs up to kMaxStages and
    // the shared-memory budget.
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
    if (range <= kTileMax) {
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
    if (p->probe_kind == SWITCHSD_PROBE_MLP) {
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
        if (launch_mlp_tc(probe_in, probe_w, part, p->B, p->d, p->probe_hidden, probe_pf, stream) != cudaSuccess)
            return SWITCHSD_ERR_CUDA;
        args.z1_part = part;
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
                            args.hidden_rows, cs != nullptr ? &ic : nullptr);
    }
    const cudaError_t e = cs ? launch_step<true>(args, split, stream) : launch_step<false>(args, split, stream);
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
