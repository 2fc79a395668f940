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
#include "step.cuh"

namespace switchsd {

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
    __shared__ int32_t s_wtot[kStepWarps];                     // candidate mode: marks per warp in a pass
    __shared__ int32_t s_choice;                               // candidate verification: the kept candidate
    __shared__ int32_t s_probe_late;                           // early probe: its copies did not land in time

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const uint32_t rank = cluster_ctarank();
    const uint32_t C = cluster_nctarank();
    // The leader is the last CTA: its range holds the most recent ends, so the candidate mode finds
    // most continuations in its own staged tile.
    const uint32_t lead = C - 1;
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
        if (rank == lead) {
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
                // Slot 0 is read before the count arrives (every row uses it unless the count is bad),
                // so a row with at most one candidate -- a neural draft -- waits for one round trip.
                if (w == 0 || w < ncx) {
                    const size_t o = size_t(b) * a.W + w;
                    const int32_t *c = a.pv_draft + o * a.D;
                    const int32_t *t = a.pv_target + o * (a.D + 1);
                    const int32_t c_lo = lane < a.D ? c[lane] : 0, c_hi = lane + 32 < a.D ? c[lane + 32] : 0;
                    const int32_t t_lo = lane < a.D ? t[lane] : 0, t_hi = lane + 32 < a.D ? t[lane + 32] : 0;
                    const int32_t len_w = a.pv_cand_len[o];
                    if (w >= ncx) break;  // warp-uniform: a bad count uses no slot
                    const int32_t len = nc > 0 ? len_w : 0;
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
    // With n_min >= 2 a match must cover the last two tokens, so the filter tests both (exact: the
    // back-compare then starts at m = 2) -- unless, in candidate mode, a candidate needs only one
    // (kappa = 1).  m0 is the length the filter has already checked.
    const int32_t kappa_c = a.kappa > 0 ? a.kappa : n_min;  // candidate mode: the gate length
    const bool pair = n_min >= 2 && (!kCand || kappa_c >= 2);
    const int32_t m0 = pair ? 2 : 1;
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
        // The early probe's partition of the slice (warps 2-7, the same order), so the logit does not
        // depend on whether the probe ran before or after the wait.
        if (warp >= 2) {
            if (probe_in)
                for (int i = tid - 2 * kWarp; i < v_staged; i += kStepThreads - 2 * kWarp)
                    zp = dot8_bf16(s_pw[i], s_ph[i], zp);
            for (int v = v0 + v_staged + tid - 2 * kWarp; v < v1; v += kStepThreads - 2 * kWarp)
                zp = dot8_bf16(__ldg(w4 + v), __ldg(h4 + v), zp);
        }
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
    if (kCand) {
        // The CTA's most recent marked ends: kStepThreads bitmap words per pass from the top; thread t
        // holds word top - t, and prefix sums of the popcounts (within the warp, then over the warps)
        // rank its bits after those of higher words.  `found` is CTA-uniform.
        const uint32_t *bm = reinterpret_cast<const uint32_t *>(tiles + a.stages * stage_ints);
        int found = 0;
        for (int top = a.bm_words - 1; top >= 0 && found < a.W; top -= kStepThreads) {
            const int idx = top - tid;
            const uint32_t wd = (idx >= 0 && !bad) ? bm[idx] : 0u;
            const int c = __popc(wd);
            int incl = c;
#pragma unroll
            for (int o = 1; o < kWarp; o <<= 1) {
                const int t = __shfl_up_sync(kFull, incl, o);
                if (lane >= o) incl += t;
            }
            if (lane == kWarp - 1) s_wtot[warp] = incl;
            __syncthreads();
            int before = found, total = 0;
#pragma unroll
            for (int w = 0; w < kStepWarps; ++w) {
                before += w < warp ? s_wtot[w] : 0;
                total += s_wtot[w];
            }
            int r = before + incl - c;
            uint32_t w2 = wd;
            while (w2 != 0u && r < a.W) {
                const int bit = 31 - __clz(w2);
                w2 &= ~(1u << bit);
                s_cand[r++] = e_lo + idx * 32 + bit;
            }
            found += total;
            __syncthreads();  // s_wtot is rewritten by the next pass
        }
        if (tid == 0) s_ncand = found < a.W ? found : a.W;
    }
    __syncthreads();
    float cta_z = 0.f;
    if (warp == 0) cta_z = warp_sum_f32(lane < kStepWarps ? s_wz[lane] : 0.f);

    // Every CTA has started and read ctx_lens[b] once this returns (they all arrived long ago).
    cluster_wait_acquire();
    if (rank == lead && verifying) {
        // The leader publishes the append; the other CTAs only patched their staged copies.
        for (int i = tid; i <= acc; i += kStepThreads) row[L_old + i] = s_app[i];
        if (tid == 0 && len_ok) {
            a.lens[b] = L;
            a.out_accept[b] = acc;
        }
    }

    // Ship this CTA's message to the leader: asynchronous DSMEM stores that complete on its barrier.
    const uint32_t done_addr = map_to_rank(&s_done, lead);
    if (tid == 0) {
        uint4 h;
        h.x = uint32_t(best & 0xffffffffu);
        h.y = uint32_t(best >> 32);
        h.z = __float_as_uint(cta_z);
        h.w = kCand ? uint32_t(s_ncand) : 0u;
        st_async_v4(map_to_rank(&s_slot[rank], lead), h, done_addr);
    } else if (tid <= kwords) {
        const uint4 v = kCand ? *reinterpret_cast<const uint4 *>(&s_cand[4 * (tid - 1)])
                              : *reinterpret_cast<const uint4 *>(&s_mine[4 * (tid - 1)]);
        st_async_v4(map_to_rank(&s_slot[rank].cand[4 * (tid - 1)], lead), v, done_addr);
    }
    if (rank != lead) return;

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
            // lane r holds CTA r's count; a suffix sum over the lanes places its ends after those of the
            // more recent CTAs r+1 .. C-1; then lanes copy (CTA, end) pairs in parallel.
            const int cnt = (hit && uint32_t(lane) < C) ? min(int(s_slot[lane].count), a.W) : 0;
            int incl = cnt;
#pragma unroll
            for (int o = 1; o < kWarp; o <<= 1) {
                const int t = __shfl_down_sync(kFull, incl, o);
                if (lane + o < kWarp) incl += t;
            }
            const int off = incl - cnt;
            for (int j0 = 0; j0 < int(C) * kMaxCand; j0 += kWarp) {  // warp-uniform bound
                const int j = j0 + lane;
                const int r = min(j / kMaxCand, int(C) - 1), i = j - r * kMaxCand;
                const int cnt_r = __shfl_sync(kFull, cnt, r);
                const int off_r = __shfl_sync(kFull, off, r);
                if (j < int(C) * kMaxCand && i < cnt_r && off_r + i < a.W) s_cand[off_r + i] = s_slot[r].cand[i];
            }
            __syncwarp();
            ncand = min(__shfl_sync(kFull, incl, 0), a.W);
        }
        const bool gate = kCand ? ncand > 0 : n >= kappa;
        int32_t mode = SWITCHSD_MODE_NO_REP;
        if (hit) mode = (gate && z >= a.logit_tau) ? SWITCHSD_MODE_COPY : SWITCHSD_MODE_REP_NO_COPY;
        const int32_t len = (!kCand && mode == SWITCHSD_MODE_COPY) ? min(a.k, L - 1 - e) : 0;
        if (lane == 0) {
            s_out[0] = int32_t(win);
            s_out[1] = len;
            if (kCand) s_ncand = mode == SWITCHSD_MODE_COPY ? ncand : 0;
            if (!kCand && a.counters)  // out_mode still holds the previous step's mode
                count_row(a.counters, mode, verifying, a.out_mode[b], s_ver[0]);
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
        // The candidates' continuations: from the leader's own staged tile for ends in its range (one
        // stage: it holds the range, its look-ahead and the patched append), else from the row (the
        // leader's append is visible to its threads after the barrier).
        const int nc = s_ncand;
        if (tid == 0) a.out_ncand[b] = nc;
        const bool one_stage = ntiles == 1;
        const int32_t off0 = kHalo - e_lo;  // tiles[off0 + p] = x[p] over the staged range
        for (int t = tid; t < nc * a.D; t += kStepThreads) {
            const int w = t / a.D, i = t - w * a.D;
            const int32_t ew = s_cand[w];
            const int32_t lw = min(a.D, L - 1 - ew);
            if (i == 0) a.out_cand_len[size_t(b) * a.W + w] = lw;
            if (i < lw) {
                const int32_t p = ew + 1 + i;
                a.out_cand[(size_t(b) * a.W + w) * a.D + i] =
                    (one_stage && ew >= e_lo && ew < e_hi) ? tiles[off0 + p] : row[p];
            }
        }
    }
}

// ------------------------------------------------------------------------------------------------
// Launch.
// ------------------------------------------------------------------------------------------------
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

cudaError_t launch_step_kernel(const StepArgs &args, bool cand, int split, cudaStream_t stream) {
    return cand ? launch_step<true>(args, split, stream) : launch_step<false>(args, split, stream);
}

}  // namespace switchsd
