// rescan.cu -- the rescan kernel: switchsd_step / switchsd_verify_step / switchsd_verify_sampled_step and the
// candidate entry points, with the linear probe (Eq. 3) or the two-layer probe's finish, laid out for a
// short chain of dependent phases after the grid-dependency wait.
//
// Paper: §3.3 (kappa-gram gate, recency-ranked copy candidates, Eq. 4 decision rule, parallel
// verification), Eq. 3 (linear probe), Fig. 1 (three cases).
//
// Row b is handled by a cluster of C CTAs of kRescanThreads threads (grid = C x B).  The row's old
// candidate ends [0, L_old - 1) are split into C contiguous 16-byte-aligned ranges; each CTA stages its
// range (plus kHalo tokens of look-back and kFwd of look-ahead) with one bulk copy, and the row's last
// kHalo tokens with another, as soon as it has read the row length -- before the grid-dependency wait
// when the caller allows it -- and, in the hash instance, warps 1.. hash every staged old end into one
// byte once the copy lands.  The CTAs are small (four warps, at most 64 registers a thread) so that the
// next launch's CTAs are resident, with their copies in flight, while this launch finishes.
//
// After the wait no cluster-wide barrier is on the path, and no CTA-wide one outside candidate mode
// (the hash instance's barrier on the hash bytes completes before the wait when the context is
// prefetched):
//  * every warp verifies the previous draft itself (the draft and the target are a few L2 lines), and
//    keeps its own window of the row's last kHalo old tokens followed by the appended tokens: the new
//    suffix and the appended positions come from it, so the staged tile is never patched;
//  * every warp scans its share of the CTA's old ends (a hash filter on the last F tokens -- computed
//    from the tokens, or the pre-wait hash bytes -- then an exact test and a backward compare against
//    its suffix window), and the leader's warp 0 also tests the a+1 ends the append creates;
//  * every warp ships its best key, its share of the probe's dot product and its best match's
//    continuation (from the staged tile, or from its window past the old length) to the row's leader CTA
//    (the last one) with asynchronous DSMEM stores completing on the leader's mbarrier, and is done.
// The leader's warp 0 publishes the append, waits (bounded) for the C x kRescanWarps messages, reduces
// them in a fixed order and writes the outputs.  The only cluster barrier is arrived on right after the
// length read and waited on just before the first message, so the leader's message barrier is
// initialised before anyone ships to it and no CTA reads the length after the leader rewrites it.
#include <mutex>

#include "mlp.cuh"
#include "step.cuh"

namespace switchsd {

// Per-warp window of y = old context followed by the append: s_y[w][j] = y[L_old - kHalo + j].
constexpr int kYLen = kHalo + SWITCHSD_KMAX + 4;
// 32-bit match keys: m << kKeyShift | e with m <= SWITCHSD_NMAX (bits 25..30) and e < 2^25; bit 31 alone
// marks a copy that did not land.
constexpr int kKeyShift = 25;
constexpr uint32_t kKeyEndMask = (1u << kKeyShift) - 1u;
constexpr uint32_t kKeyTimeout = 1u << 31;
static_assert(SWITCHSD_NMAX < (1 << (31 - kKeyShift)), "m must fit below the timeout bit");
// The scan: kScanWords words per thread per round; a thread's rounds of a CTA range fit the 32 bits of its
// pass mask.
constexpr int kScanWords = 4;
static_assert(kRescanTileMax / 4 / (kScanWords * kRescanThreads) <= 32, "a thread's rounds fit its pass mask");

// The scan of a CTA's old ends [e_lo, e_end) against the new suffix (suf[-q] = its q-th token from the end)
// for the longest-then-most-recent match: the largest key m << kKeyShift | e over the ends with
// m(e) >= n_min, 0 if none.  stage[kHalo + p - e_lo] = x[p] over [e_lo - kHalo, e_end + kFwd).
//
// Filter depth F = min(n_min, 3): end e can match only if its last F tokens equal the suffix's.  Pass 1
// tests a hash of them, h(e) = x[e] + x[e-1] A + x[e-2] B (the first F terms, mod 2^32), against the
// suffix's: equal tokens give equal hashes, so no end that matches is missed, and the few that collide
// are dropped by pass 2's exact test.  Two multiply-adds per end and a running three-input min test a
// round of sixteen ends; the shared-memory reads, not the arithmetic, set the pace.
//
// Pass 1: rounds of kScanWords words per thread (word g0 + u kT, g0 = tid + kScanWords kT r: consecutive
// lanes read consecutive words), each with the two tokens before it (unset before position 0, where
// lim < F drops the end); a round with an end that passes only sets its bit.  No branch and no backward
// compare in the hot loop.
// Pass 2 (rare): the rounds that passed, in warp-synchronous steps (each step every lane with a round left
// takes its next one, so the compares of a hot suffix run side by side), reloaded from shared memory;
// their ends that pass the exact test (x[e-i] = suf[-i] for i < F) take the backward compare from m = F,
// eight positions per step with independent loads.
constexpr uint32_t kHashA = 0x9E3779B1u, kHashB = 0x85EBCA77u;  // odd multipliers

// The F-token hash of end e (x0 = x[e], x1 = x[e-1], x2 = x[e-2]; the first F terms, mod 2^32).
template <int F>
__device__ __forceinline__ uint32_t end_hash(int32_t x0, int32_t x1, int32_t x2) {
    uint32_t h = uint32_t(x0);
    if (F >= 2) h += uint32_t(x1) * kHashA;
    if (F >= 3) h += uint32_t(x2) * kHashB;
    return h;
}
// One byte of it for the pre-wait table (multiplicative: the top byte of an odd multiple).
__device__ __forceinline__ uint32_t hash_byte(uint32_t h) { return (h * 0x2C1B3C6Du) >> 24; }
// Nonzero iff some byte of v is zero (exact as a whole-word test).
__device__ __forceinline__ uint32_t has_zero_byte(uint32_t v) { return (v - 0x01010101u) & ~v & 0x80808080u; }

// Pre-wait hashing: hb[g] holds the hash bytes of the ends e_lo + 4g .. + 3 (byte j = end e_lo + 4g + j),
// for the words g < n4 of this CTA's old ends; threads t, t + nt, ... of the caller take one word each.
template <int F>
__device__ __forceinline__ void hash_ends(const int32_t *stage, uint32_t *hb, int32_t n4, int t, int nt) {
    const int4 *g4 = reinterpret_cast<const int4 *>(stage + kHalo);
    for (int32_t g = t; g < n4; g += nt) {
        const int4 v = g4[g];
        const int2 pv = F >= 2 ? *reinterpret_cast<const int2 *>(stage + kHalo + 4 * g - 2) : make_int2(0, 0);
        hb[g] = hash_byte(end_hash<F>(v.x, pv.y, pv.x)) | hash_byte(end_hash<F>(v.y, v.x, pv.y)) << 8 |
                hash_byte(end_hash<F>(v.z, v.y, v.x)) << 16 | hash_byte(end_hash<F>(v.w, v.z, v.y)) << 24;
    }
}

//
// Candidate mode (kCand): every end whose common suffix reaches kappa_c is also marked in the CTA's bitmap
// bm (bit e - e_lo; F <= kappa_c, so the filter passes every such end).
//
// kPre: the hashes were taken before the grid-dependency wait (hash_ends into hb); pass 1 then compares
// one byte per end against the suffix's (four ends a 4-byte load), and pass 2 takes only the ends whose
// byte matches.  The byte filter passes every end that matches and about 1 in 256 of the others, which
// the exact test drops.
template <int F, bool kCand, bool kPre>
__device__ __forceinline__ uint32_t scan_ends(const int32_t *stage, int32_t e_lo, int32_t e_end, const int32_t *suf,
                                              int32_t n_min, int32_t n_max, int tid, int lane,
                                              uint32_t *bm = nullptr, int32_t kappa_c = 0,
                                              const uint32_t *hb = nullptr) {
    const int32_t s0 = suf[0], s1 = F >= 2 ? suf[-1] : 0, s2 = F >= 3 ? suf[-2] : 0;
    const uint32_t hs = end_hash<F>(s0, s1, s2);
    const uint32_t hs4 = hash_byte(hs) * 0x01010101u;
    const int32_t n4 = (e_end - e_lo + 3) >> 2;
    const int4 *g4 = reinterpret_cast<const int4 *>(stage + kHalo);
    const int32_t off = kHalo - e_lo;
    uint32_t passed = 0u;
    int rnd = 0;
    if constexpr (kPre) {
        for (int32_t g0 = tid; g0 - lane < n4; g0 += kScanWords * kRescanThreads, ++rnd) {
            uint32_t z = 0u;
#pragma unroll
            for (int u = 0; u < kScanWords; ++u) {
                const int32_t g = g0 + u * kRescanThreads;
                z |= g < n4 ? has_zero_byte(hb[g] ^ hs4) : 0u;
            }
            passed |= uint32_t(z != 0u) << (rnd & 31);
        }
    } else {
        auto hash = [&](int32_t x0, int32_t x1, int32_t x2) { return end_hash<F>(x0, x1, x2) ^ hs; };
        for (int32_t g0 = tid; g0 - lane < n4; g0 += kScanWords * kRescanThreads, ++rnd) {
            int4 v[kScanWords];
            int2 pv[kScanWords];  // x[4g - 2], x[4g - 1]
#pragma unroll
            for (int u = 0; u < kScanWords; ++u) {
                const int32_t g = g0 + u * kRescanThreads;
                v[u] = g < n4 ? g4[g] : make_int4(0, 0, 0, 0);
                pv[u] = (F >= 2 && g < n4) ? *reinterpret_cast<const int2 *>(stage + kHalo + 4 * g - 2) : make_int2(0, 0);
            }
            uint32_t mn = 0xffffffffu;
#pragma unroll
            for (int u = 0; u < kScanWords; ++u) {
                const uint32_t h0 = hash(v[u].x, pv[u].y, pv[u].x), h1 = hash(v[u].y, v[u].x, pv[u].y);
                const uint32_t h2 = hash(v[u].z, v[u].y, v[u].x), h3 = hash(v[u].w, v[u].z, v[u].y);
                mn = __vimin3_u32(mn, __vimin3_u32(h0, h1, h2), h3);
            }
            passed |= uint32_t(mn == 0u) << (rnd & 31);
        }
    }
    uint32_t mine = 0u;
    // m(e) from F for an end whose last F tokens match: x[e - q] against suf[-q], eight positions per step,
    // every load issued unconditionally (q clamped to lim - 1; the sentinel bit ends the run at the count)
    auto match_len = [&](int32_t e, int32_t lim) {
        int32_t m = F;
#pragma unroll 1
        while (m < lim) {
            const int32_t cnt = min(8, lim - m);
            unsigned miss = 1u << cnt;
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const int32_t q = min(m + i, lim - 1);
                miss |= unsigned(stage[off + e - q] != suf[-q]) << i;
            }
            const int32_t run = __ffs(miss) - 1;
            m += run;
            if (run < cnt) break;
        }
        return m;
    };
    auto take = [&](int32_t e, int32_t m) {
        if (m >= n_min) {
            const uint32_t key = (uint32_t(m) << kKeyShift) | uint32_t(e);
            mine = key > mine ? key : mine;
        }
        if (kCand && m >= kappa_c) atomicOr(&bm[(e - e_lo) >> 5], 1u << ((e - e_lo) & 31));
    };
    while (__any_sync(kFull, passed != 0u)) {
        if (passed == 0u) continue;
        const int r = __ffs(passed) - 1;
        passed &= passed - 1u;
        if constexpr (kPre) {
            // the round's ends whose hash byte matches: bit 4u + j for end j of word u
            uint32_t cand = 0u;
#pragma unroll
            for (int u = 0; u < kScanWords; ++u) {
                const int32_t g = tid + r * kScanWords * kRescanThreads + u * kRescanThreads;
                const uint32_t eq = g < n4 ? __vcmpeq4(hb[g], hs4) : 0u;  // 0xff in each matching byte
                cand |= ((eq & 1u) | (eq >> 7 & 2u) | (eq >> 14 & 4u) | (eq >> 21 & 8u)) << (4 * u);
            }
            while (cand) {
                const int i = __ffs(cand) - 1;
                cand &= cand - 1u;
                const int32_t g = tid + r * kScanWords * kRescanThreads + (i >> 2) * kRescanThreads;
                const int32_t e = e_lo + 4 * g + (i & 3);
                if (e >= e_end) break;
                const int32_t lim = min(n_max, e + 1);
                if (lim < F) continue;  // the hash read a token before position 0
                bool ok = stage[off + e] == s0;
                if (F >= 2) ok = ok && stage[off + e - 1] == s1;
                if (F >= 3) ok = ok && stage[off + e - 2] == s2;
                if (ok) take(e, match_len(e, lim));
            }
        } else {
#pragma unroll 1
            for (int u = 0; u < kScanWords; ++u) {
                const int32_t g = tid + r * kScanWords * kRescanThreads + u * kRescanThreads;
                if (g >= n4) break;
                const int4 v = g4[g];
                const int2 pv = *reinterpret_cast<const int2 *>(stage + kHalo + 4 * g - 2);
                // exact test of the last F tokens of each end
                const int32_t x[6] = {pv.x, pv.y, v.x, v.y, v.z, v.w};
                uint32_t hall = 0u;
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    bool ok = x[j + 2] == s0;
                    if (F >= 2) ok = ok && x[j + 1] == s1;
                    if (F >= 3) ok = ok && x[j] == s2;
                    hall |= uint32_t(ok) << j;
                }
                while (hall) {
                    const int j = __ffs(hall) - 1;
                    hall &= hall - 1;
                    const int32_t e = e_lo + 4 * g + j;
                    if (e >= e_end) break;
                    const int32_t lim = min(n_max, e + 1);
                    if (lim < F) continue;  // the test read a token before position 0
                    take(e, match_len(e, lim));
                }
            }
        }
    }
    return mine;
}

constexpr int kVerifyLoads = 4;  // candidate verification: staging loads a thread has in flight at once

// Candidate mode's shared memory beyond the single-draft layout: per CTA one candidate message of cslot
// bytes -- a 16-byte header (count), the ends (W, most recent first), their continuations [W][D] -- the
// leader receiving C of them and every CTA staging its own; a bitmap of the CTA's marked ends; the
// verification's staging of the previous candidates (drafts [W][D], targets [W][D+1], lengths [W], count).
struct CandLayout {
    uint32_t cslot;  // bytes of a candidate message
    int bm_words;    // bitmap words (a multiple of 4)
    int v_ints;      // verification staging (a multiple of 4)
};
__host__ __device__ inline CandLayout cand_layout(int tile, int W, int D) {
    CandLayout c;
    c.cslot = 16u * uint32_t(1 + (W + 3) / 4 + (W * D + 3) / 4);
    c.bm_words = ((tile + 31) / 32 + 3) & ~3;
    c.v_ints = (W * D + W * (D + 1) + W + 1 + 3) & ~3;
    return c;
}

// kPre: the pre-wait hash table (a.hash_words > 0); kMlp: the two-layer probe's finish (a.z1_part set).
// Separate instances, so that each carries only its own scan and its own probe code and registers.
template <bool kSampled, bool kCand, bool kPre, bool kMlp>
__global__ void __launch_bounds__(kRescanThreads, kRescanLaunchBlocks) rescan_kernel(const StepArgs a) {
    extern __shared__ __align__(128) int32_t dsm[];
    __shared__ __align__(8) uint64_t bars[5];              // tile, tail, probe slices, messages (leader),
                                                           // pre-wait hashes
    __shared__ __align__(16) int32_t s_tail[kHalo + 8];    // x[tail_lo .. L_old), tail_lo = roundown4(L_old - kHalo)
    __shared__ int32_t s_y[kRescanWarps][kYLen];
    __shared__ int32_t s_sel[kMaxCand];                    // candidate mode: the CTA's selected ends / the
                                                           // leader's merged candidates' sources
    __shared__ int32_t s_wtot[kRescanWarps];               // candidate mode: marks per warp in a pass

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const uint32_t rank = cluster_ctarank();
    const uint32_t C = cluster_nctarank();
    const uint32_t lead = C - 1;
    const int b = blockIdx.y;
    const int stage_ints = kHalo + a.tile + kFwd;
    int32_t *stage = dsm;
    uint32_t *hb = reinterpret_cast<uint32_t *>(dsm + ((stage_ints + 3) & ~3));  // [hash_words]
    uint4 *s_pw = reinterpret_cast<uint4 *>(hb + a.hash_words);
    uint4 *s_ph = s_pw + a.probe_words;
    unsigned char *msgs = reinterpret_cast<unsigned char *>(s_ph + a.probe_words);
    const bool verifying = a.pv_len != nullptr;
    const int kw = kCand ? 0 : (a.k + 3) >> 2;             // 16-byte words of a message's continuation
    const uint32_t slot_bytes = 16u * uint32_t(1 + kw);
    const int nmsg = int(C) * kRescanWarps;
    const CandLayout cl = cand_layout(kCand ? a.tile : 0, kCand ? a.W : 0, kCand ? a.D : 0);
    unsigned char *cmsgs = msgs + size_t(nmsg) * slot_bytes;                  // [C][cslot] (leader)
    unsigned char *cstage = cmsgs + size_t(C) * cl.cslot;                     // this CTA's message
    uint32_t *bm = reinterpret_cast<uint32_t *>(cstage + cl.cslot);           // [bm_words]
    int32_t *vc = reinterpret_cast<int32_t *>(bm + cl.bm_words);              // previous drafts [W][D]
    int32_t *vt = vc + a.W * a.D;                                             // their targets [W][D+1]
    int32_t *vl = vt + a.W * (a.D + 1);                                       // their lengths [W]

    if (tid == 0) {
        mbar_init(&bars[0], 1);
        mbar_init(&bars[1], 1);
        mbar_init(&bars[2], 1);
        mbar_init(&bars[4], kRescanThreads - kWarp);
        if (rank == lead) {
            mbar_init(&bars[3], 1);
            mbar_arrive_expect_tx(&bars[3], slot_bytes * uint32_t(nmsg) + (kCand ? cl.cslot * C : 0u));
        }
        fence_mbar_init();
    }
    if (kCand)
        for (int i = tid; i < cl.bm_words; i += kRescanThreads) bm[i] = 0u;
    __syncthreads();  // the barriers are initialised (and the bitmap cleared) before any thread uses them

    const bool pf_ctx = (a.prefetch & SWITCHSD_PREFETCH_CONTEXT) != 0;
    const bool gather = verifying && a.hidden_rows > 1;
    // Two-layer probe: the first layer's split-K partial sums come from the probe kernel just before this
    // one (read after the wait); this CTA finishes units [u0, u1) (b1, ReLU, w2).
    constexpr bool mlp = kMlp;
    const bool pf_probe = (a.prefetch & SWITCHSD_PREFETCH_PROBE) != 0 && !gather && !mlp;
    // Two-layer probe: every input but the partial sums was written by kernels that completed before the
    // first-layer kernel released this launch (it does so only after its own wait), so verification and
    // scan run while it computes; warps 1.. wait just before reading the sums.  Reads before that wait
    // go through L2 (bulk copies, ld.global.cg).
    const bool late = mlp && a.wait_late != 0;
    if (!pf_ctx && !late) pdl_wait();
    int32_t *row = a.ctx + size_t(b) * size_t(a.cap);
    // The CTA's ends are split on the row's old length, or, with a length bound, on the bound: its tile
    // copy then leaves before the length is read, and a row longer than the bound is a bad length.
    const bool bounded = a.len_bound > 0;
    auto range_of = [&](int32_t E, int32_t &e_lo_, int32_t &e_hi_) {
        int32_t chunk = (E + int32_t(C) - 1) / int32_t(C);
        chunk = (chunk + 3) & ~3;
        e_lo_ = min(E, int32_t(rank) * chunk);
        e_hi_ = min(E, e_lo_ + chunk);
    };
    int32_t e_lo = 0, e_hi = 0, lo = 0;
    if (bounded) {
        range_of(a.len_bound - 1, e_lo, e_hi);
        lo = max(0, e_lo - kHalo);
    }
    auto tile_hi = [&]() { return e_hi > e_lo ? min((e_hi + kFwd + 3) & ~3, a.cap) : lo; };
    const uint64_t pol = l2_evict_first_policy();
    auto issue_tile = [&](int32_t hi_) {  // positions [lo, hi_) land at stage[kHalo + p - e_lo]
        const uint32_t bytes = uint32_t(hi_ - lo) * 4u;
        mbar_expect_tx_relaxed(&bars[0], bytes);
        if (bytes > 0) bulk_g2s_hint(stage + (kHalo + lo - e_lo), row + lo, bytes, &bars[0], pol);
    };
    if (bounded && tid == 0) issue_tile(tile_hi());
    // Every thread reads the length itself (one L2 request per warp), then arrives on the cluster
    // barrier.  The arrive is relaxed: the barrier only has to publish the leader's message barrier (its
    // initialisation fence is a release), and each warp's read of the length is ordered before the leader
    // rewrites it by the data itself -- the warp's message is computed from the length, and the leader
    // rewrites it only after every message has landed.
    const int32_t L_old = __ldcg(a.lens + b);
    cluster_arrive_relaxed();
    const bool len_ok = L_old >= 1 && L_old <= (bounded ? a.len_bound : a.cap);
    const int32_t E_old = len_ok ? L_old - 1 : 0;
    if (!bounded) {
        range_of(E_old, e_lo, e_hi);
        lo = max(0, e_lo - kHalo);
    }
    const int32_t hi = tile_hi();                       // the staged positions end here
    const int32_t e_end = max(e_lo, min(e_hi, E_old));  // the old ends scanned: [e_lo, e_end)
    const int32_t tail_lo = max(0, (L_old - kHalo) & ~3);
    const int32_t tail_hi = len_ok ? (L_old + 3) & ~3 : tail_lo;  // <= cap since cap % 4 == 0

    // Linear probe: this CTA's slice is words [v0, v1) of 8 bf16; the first probe_words of w and h are
    // staged by bulk copies, the rest read directly.  Warps 1.. compute it (warp 0 issues the copies and
    // releases the next launch).
    const int nv = a.d >> 3;
    const int vper = (nv + int(C) - 1) / int(C);
    const int v0 = min(nv, int(rank) * vper), v1 = min(nv, v0 + vper);
    const int v_staged = (gather || mlp) ? 0 : min(v1 - v0, a.probe_words);
    const uint4 *w4 = reinterpret_cast<const uint4 *>(a.probe_w);
    const uint4 *h4 = reinterpret_cast<const uint4 *>(a.hidden + size_t(b) * size_t(gather ? a.hidden_rows : 1) *
                                                                  size_t(a.d));
    auto issue_probe = [&]() {
        const uint32_t pb = uint32_t(v_staged) * 16u;
        mbar_expect_tx_relaxed(&bars[2], 2u * pb);
        if (pb > 0) {
            bulk_g2s(s_pw, w4 + v0, pb, &bars[2]);
            bulk_g2s(s_ph, h4 + v0, pb, &bars[2]);
        }
    };
    if (tid == 0) {
        const uint32_t tb = uint32_t(tail_hi - tail_lo) * 4u;
        mbar_expect_tx_relaxed(&bars[1], tb);
        if (tb > 0) bulk_g2s_hint(s_tail, row + tail_lo, tb, &bars[1], pol);
        if (pf_probe) issue_probe();
        if (!bounded) issue_tile(hi);
        // The parameters only the leader's last phase reads are fetched now, so that phase does not wait
        // on the constant cache.
        asm volatile("" ::"l"(a.out_mode), "l"(a.out_len), "l"(a.out_score), "l"(a.out_match_n), "l"(a.out_match_end),
                     "l"(a.status), "l"(a.out_draft), "l"(a.out_accept), "r"(a.kappa), "f"(a.logit_tau));
    }
    float zp = 0.f;
    bool probe_ok = true;
    auto probe_dot = [&](const uint4 *h) {  // warps 1..: thread j = tid - 32 takes words j, j + kT - 32, ...
        if (v_staged > 0) {
            probe_ok = mbar_wait(&bars[2], 0);
            if (probe_ok)
                for (int i = tid - kWarp; i < v_staged; i += kRescanThreads - kWarp) zp = dot8_bf16(s_pw[i], s_ph[i], zp);
        }
        for (int v = v0 + v_staged + tid - kWarp; v < v1; v += kRescanThreads - kWarp)
            zp = dot8_bf16(__ldg(w4 + v), __ldg(h + v), zp);
    };
    // A prefetched probe is finished before the wait by warps 1.. (its inputs are not written by the
    // preceding kernel); warp 0 goes straight to the wait and releases the next launch.
    if (pf_probe && warp >= 1) probe_dot(h4);
    // Warps 1.. hash this CTA's old ends once the tile has landed -- before the wait when the context is
    // prefetched -- so that the scan after it compares one byte per end (scan_ends, kPre).
    constexpr bool pre = kPre;
    // the filter depth F (in candidate mode no deeper than the gate length kappa)
    auto filter_depth = [&]() {
        return min(kCand ? min(a.n_min, a.kappa > 0 ? a.kappa : a.n_min) : a.n_min, 3);
    };
    if (pre && warp >= 1) {
        const int fdepth = filter_depth();
        if (len_ok && (hi == lo || mbar_wait(&bars[0], 0))) {
            const int32_t n4 = (e_end - e_lo + 3) >> 2;
            if (fdepth >= 3) hash_ends<3>(stage, hb, n4, tid - kWarp, kRescanThreads - kWarp);
            else if (fdepth == 2) hash_ends<2>(stage, hb, n4, tid - kWarp, kRescanThreads - kWarp);
            else hash_ends<1>(stage, hb, n4, tid - kWarp, kRescanThreads - kWarp);
        }
        mbar_arrive(&bars[4]);  // every thread of warps 1.., whether or not it hashed
    }
    if (pf_ctx && !late) pdl_wait();
    pdl_trigger();
    if (!pf_probe && !gather && !mlp && tid == 0) issue_probe();

    // Two-layer probe: this CTA finishes units [u0m, u1m) (the S partial sums in order, b1, ReLU, w2);
    // thread j = tid - 32 of warps 1.. takes units u0m + j, u0m + j + (kT - 32), ...  When this launch's
    // wait already covers the first-layer kernel (not late), the first unit's partial sums are loaded
    // now, so that their round trip overlaps the verification's; the sums are taken after it.
    const int uper = mlp ? (a.H1 + int(C) - 1) / int(C) : 0;
    const int u0m = min(a.H1, int(rank) * uper), u1m = min(a.H1, u0m + uper);
    auto mlp_unit = [&](int u, const float *pz, float acc) {
        float z1 = 0.f;
#pragma unroll
        for (int sp = 0; sp < kMaxMlpSplit; ++sp)
            if (sp < a.mlp_S) z1 += pz[sp];
        if (a.b1) z1 += a.b1[u];
        return fmaf(bf16_lo(uint32_t(a.w2[u])), fmaxf(z1, 0.f), acc);
    };
    auto mlp_load = [&](int u, float *pz) {
#pragma unroll
        for (int sp = 0; sp < kMaxMlpSplit; ++sp)
            pz[sp] = sp < a.mlp_S ? __ldcg(a.z1_part + (size_t(sp) * a.B + size_t(b)) * a.H1p + u) : 0.f;
    };
    // every partial sum of a unit is loaded before the first add (independent L2 reads), then added in
    // order; the same threads and order either way, so the logit does not depend on when this runs
    auto mlp_finish = [&](int from) {
        for (int u = from; u < u1m; u += kRescanThreads - kWarp) {
            float pz[kMaxMlpSplit];
            mlp_load(u, pz);
            zp = mlp_unit(u, pz, zp);
        }
    };
    const bool mlp_early = mlp && !late && warp >= 1;
    float pz0[kMaxMlpSplit];
    const int u_first = u0m + tid - kWarp;
    if (mlp_early && u_first < u1m) mlp_load(u_first, pz0);

    // ---- verification of the previous draft (every warp) ----
    int32_t acc = -1, L = L_old, vst = len_ok ? SWITCHSD_ROW_OK : SWITCHSD_ROW_BAD_LEN;
    int32_t d_lo = 0, d_hi = 0, t_acc = 0;
    int32_t choice = 0;  // candidate mode: the kept candidate
    if (kCand && verifying) {
        // The W previous candidates verified at once (§3.3): the CTA stages every slot's draft, target and
        // length (one round of independent L2 reads, whatever the count), then each warp takes, per
        // candidate, the first position where draft and target differ; the longest accepted candidate is
        // kept, the lowest index on a tie.  A count of 0 (a neural draft) uses slot 0 with length 0.
        const int W = a.W, D = a.D;
        const size_t o = size_t(b) * size_t(W);
        // one index space over drafts, targets, lengths and the count (vl[W]); each thread issues all of
        // its loads before its first store, so they share one round trip
        const int n_d = W * D, n_t = W * (D + 1), n_all = n_d + n_t + W + 1;
        for (int base = tid; base < n_all; base += kVerifyLoads * kRescanThreads) {
            int32_t v[kVerifyLoads];
#pragma unroll
            for (int u = 0; u < kVerifyLoads; ++u) {
                const int i = base + u * kRescanThreads;
                v[u] = 0;
                if (i < n_d) v[u] = __ldcg(a.pv_draft + o * D + i);
                else if (i < n_d + n_t) v[u] = __ldcg(a.pv_target + o * (D + 1) + (i - n_d));
                else if (i < n_d + n_t + W) v[u] = __ldcg(a.pv_cand_len + o + (i - n_d - n_t));
                else if (i < n_all) v[u] = __ldcg(a.pv_len + b);
            }
#pragma unroll
            for (int u = 0; u < kVerifyLoads; ++u)
                if (base + u * kRescanThreads < n_all) vc[base + u * kRescanThreads] = v[u];  // vc, vt, vl contiguous
        }
        __syncthreads();
        const int32_t nc = vl[W];
        if (len_ok) {
            bool badlen = nc < 0 || nc > W;
            const int ncx = badlen ? 0 : (nc > 0 ? nc : 1);
            int32_t best = -1, best_w = 0;
            for (int w = 0; w < ncx; ++w) {
                const int32_t len = nc > 0 ? vl[w] : 0;
                badlen |= len < 0 || len > D;
                const int32_t lc = (len >= 0 && len <= D) ? len : 0;
                const int32_t *cw_ = vc + w * D, *tw_ = vt + w * (D + 1);
                const unsigned m_lo = __ballot_sync(kFull, lane < lc && cw_[lane] != tw_[lane]);
                const unsigned m_hi = __ballot_sync(kFull, lane + 32 < lc && cw_[lane + 32] != tw_[lane + 32]);
                const int32_t acc_w = m_lo ? __ffs(m_lo) - 1 : (m_hi ? 32 + __ffs(m_hi) - 1 : lc);
                if (acc_w > best) {
                    best = acc_w;
                    best_w = w;
                }
            }
            choice = best_w;
            if (badlen) {
                vst = SWITCHSD_ROW_BAD_LEN;
            } else if (L_old + best + 1 > a.cap) {
                vst = SWITCHSD_ROW_CAPACITY;
            } else {
                acc = best;
                L = L_old + acc + 1;
            }
        }
    }
    if (!kCand && verifying && len_ok) {
        const int32_t *dr = a.pv_draft + size_t(b) * a.k;
        const int32_t *tg = a.pv_target + size_t(b) * (a.k + 1);
        const int32_t pv_n = __ldcg(a.pv_len + b);
        d_lo = lane < a.k ? __ldcg(dr + lane) : 0;
        d_hi = lane + 32 < a.k ? __ldcg(dr + lane + 32) : 0;
        const int32_t t_lo = lane <= a.k ? __ldcg(tg + lane) : 0;
        const int32_t t_hi = lane + 32 <= a.k ? __ldcg(tg + lane + 32) : 0;
        const int32_t t_top = (lane == 0 && a.k >= 64) ? __ldcg(tg + 64) : 0;
        if (pv_n < 0 || pv_n > a.k) {
            vst = SWITCHSD_ROW_BAD_LEN;
        } else {
            bool rej_lo, rej_hi;
            if (kSampled) {
                // T > 0: draft token i is rejected when u_i * q_i (binary32) is not below p_i
                const size_t o = size_t(b) * a.k;
                rej_lo = lane < pv_n && !(__fmul_rn(__ldcg(a.pv_u + o + lane), a.pv_q ? __ldcg(a.pv_q + o + lane) : 1.f) <
                                          __ldcg(a.pv_p + o + lane));
                rej_hi = lane + 32 < pv_n &&
                         !(__fmul_rn(__ldcg(a.pv_u + o + lane + 32), a.pv_q ? __ldcg(a.pv_q + o + lane + 32) : 1.f) <
                           __ldcg(a.pv_p + o + lane + 32));
            } else {
                rej_lo = lane < pv_n && d_lo != t_lo;
                rej_hi = lane + 32 < pv_n && d_hi != t_hi;
            }
            const unsigned m_lo = __ballot_sync(kFull, rej_lo);
            const unsigned m_hi = __ballot_sync(kFull, rej_hi);
            const int32_t at = m_lo ? __ffs(m_lo) - 1 : (m_hi ? 32 + __ffs(m_hi) - 1 : pv_n);
            if (L_old + at + 1 > a.cap) {
                vst = SWITCHSD_ROW_CAPACITY;
            } else {
                acc = at;
                t_acc = __shfl_sync(kFull, acc < 32 ? t_lo : (acc < 64 ? t_hi : t_top), acc & 31);
                L = L_old + acc + 1;
            }
        }
    }
    if (mlp_early && u_first < u1m) {
        zp = mlp_unit(u_first, pz0, zp);
        mlp_finish(u_first + (kRescanThreads - kWarp));
    }
    // The probed state of a fused verification with hidden_rows = k + 1: row a_b (row 0 when nothing was
    // appended).  Its words are loaded now and used after the scan.
    uint4 gw = make_uint4(0, 0, 0, 0), gh = make_uint4(0, 0, 0, 0);
    if (gather) {
        h4 += size_t(acc > 0 ? acc : 0) * size_t(nv);
        const int v = v0 + tid - kWarp;
        if (warp >= 1 && v < v1) {
            gw = __ldg(w4 + v);
            gh = __ldg(h4 + v);
        }
    }

    // ---- this warp's window: y[L_old - kHalo + j], the old tail then the appended tokens ----
    const bool tail_in = tail_hi == tail_lo || mbar_wait(&bars[1], 0);
    int32_t *y = s_y[warp];
    {
        const int32_t p = L_old - kHalo + lane;
        y[lane] = (len_ok && p >= 0 && tail_in) ? s_tail[p - tail_lo] : 0;
        if (acc >= 0) {
            if (kCand) {  // the kept candidate's accepted tokens, then its target's next token
                for (int i = lane; i < acc; i += kWarp) y[kHalo + i] = vc[choice * a.D + i];
                if (lane == 0) y[kHalo + acc] = vt[choice * (a.D + 1) + acc];
            } else {
                if (lane < acc) y[kHalo + lane] = d_lo;
                if (lane + 32 < acc) y[kHalo + 32 + lane] = d_hi;
                if (lane == 0) y[kHalo + acc] = t_acc;
            }
        }
    }
    __syncwarp();
    const int32_t *suf = y + kHalo + acc;  // suf[-m] = the m-th token from the end of the new context
    const int32_t n_max = a.n_max, n_min = a.n_min;

    // ---- scan of this warp's share of the CTA's old ends ----
    const int32_t kappa_c = a.kappa > 0 ? a.kappa : a.n_min;  // candidate mode: the gate length
    uint32_t new_c[3] = {0u, 0u, 0u};                         // candidate mode: appended ends (leader)
    // key = m << kKeyShift | e (e < 2^kKeyShift, m <= 32): the largest key is the longest match, then the
    // most recent; 0 = no match; kKeyTimeout marks a copy that did not land.
    uint32_t mine = 0;
    const bool tile_in = hi == lo || mbar_wait(&bars[0], 0);
    const bool hashed = !pre || mbar_wait(&bars[4], 0);
    bool timed_out = !tail_in || !tile_in || !hashed;
    const int32_t off = kHalo - e_lo;  // stage[off + p] = x[p] over the staged range
    if (!timed_out && len_ok && L >= 2) {
        // (n_min and kappa are uniform over the launch: one instance runs)
        // the filter depth may test no more than a candidate needs (fdepth <= kappa in candidate mode)
        const int fdepth = filter_depth();
        mine = fdepth >= 3 ? scan_ends<3, kCand, kPre>(stage, e_lo, e_end, suf, n_min, n_max, tid, lane, bm, kappa_c, hb)
                           : (fdepth == 2
                                  ? scan_ends<2, kCand, kPre>(stage, e_lo, e_end, suf, n_min, n_max, tid, lane, bm, kappa_c, hb)
                                  : scan_ends<1, kCand, kPre>(stage, e_lo, e_end, suf, n_min, n_max, tid, lane, bm, kappa_c, hb));
        // The ends the append creates, [L_old - 1, L - 1), lie in the window: the leader's warp 0.  In
        // candidate mode new_c[t] bit i marks end L_old - 1 + 32 t + i as a candidate (warp-uniform).
        if (kCand && rank == lead && warp == 0 && acc >= 0) {
#pragma unroll 1
            for (int t = 0; 32 * t <= acc; ++t) {
                const int32_t j = lane + 32 * t;
                bool qual = false;
                if (j <= acc) {
                    const int32_t e = L_old - 1 + j;
                    const int32_t lim = min(n_max, e + 1);
                    int32_t m = 0;
#pragma unroll 1
                    while (m < lim && y[kHalo - 1 + j - m] == suf[-m]) ++m;
                    if (m >= n_min) {
                        const uint32_t key = (uint32_t(m) << kKeyShift) | uint32_t(e);
                        mine = key > mine ? key : mine;
                    }
                    qual = m >= kappa_c;
                }
                new_c[t] = __ballot_sync(kFull, qual);
            }
        } else if (rank == lead && warp == 0 && acc >= 0) {
#pragma unroll 1
            for (int32_t j = lane; j <= acc; j += kWarp) {
                const int32_t e = L_old - 1 + j;
                const int32_t lim = min(n_max, e + 1);
                int32_t m = 0;
#pragma unroll 1
                while (m < lim && y[kHalo - 1 + j - m] == suf[-m]) ++m;
                if (m >= n_min) {
                    const uint32_t key = (uint32_t(m) << kKeyShift) | uint32_t(e);
                    mine = key > mine ? key : mine;
                }
            }
        }
    }
    uint32_t key = __reduce_max_sync(kFull, mine);
    if (timed_out) key = kKeyTimeout;

    // ---- candidate mode: this CTA's W most recent marked ends and their continuations (warp 0) ----
    if constexpr (kCand) {
        __syncthreads();  // every warp's marks are in the bitmap
        // Bitmap words from the top, kRescanThreads per pass: thread t holds word top - t; prefix sums of
        // the popcounts (within the warp, then over the warps) rank its bits after those of higher words.
        // `found` is CTA-uniform.
        const int nwords = (e_end - e_lo + 31) >> 5;
        int found = 0;
        for (int top = nwords - 1; top >= 0 && found < a.W; top -= kRescanThreads) {
            const int idx = top - tid;
            const uint32_t wd = idx >= 0 ? bm[idx] : 0u;
            const int c = __popc(wd);
            int incl = c;
#pragma unroll
            for (int o_ = 1; o_ < kWarp; o_ <<= 1) {
                const int t_ = __shfl_up_sync(kFull, incl, o_);
                if (lane >= o_) incl += t_;
            }
            if (lane == kWarp - 1) s_wtot[warp] = incl;
            __syncthreads();
            int r = found, total = 0;
#pragma unroll
            for (int w = 0; w < kRescanWarps; ++w) {
                r += w < warp ? s_wtot[w] : 0;
                total += s_wtot[w];
            }
            r += incl - c;
            uint32_t w2 = wd;
            while (w2 != 0u && r < a.W) {
                const int bit = 31 - __clz(w2);
                w2 &= ~(1u << bit);
                s_sel[r++] = e_lo + idx * 32 + bit;
            }
            found += total;
            __syncthreads();  // s_wtot is rewritten by the next pass; s_sel is complete after the last
        }
        if (warp == 0) {
            const int nsel = min(found, a.W);
            // the message: header (count), the ends, then candidate w's D tokens at w D -- from the staged
            // tile, or past the old length from this warp's window (an end e continues for
            // min(D, L - 1 - e) tokens, all below L)
            int32_t *ce = reinterpret_cast<int32_t *>(cstage + 16);
            int32_t *ct = reinterpret_cast<int32_t *>(cstage + 16 + 16 * ((a.W + 3) / 4));
            if (lane == 0) *reinterpret_cast<int4 *>(cstage) = make_int4(nsel, 0, 0, 0);
            if (lane < nsel) ce[lane] = s_sel[lane];
            const int dw = kWarp / a.D, di = kWarp - dw * a.D;  // (candidate, token) step of 32 slots
            int w = lane / a.D, i = lane - w * a.D;
            for (int t = lane; t < nsel * a.D; t += kWarp) {
                const int32_t ew = s_sel[w];
                const int32_t p = ew + 1 + i;
                ct[t] = i < min(a.D, L - 1 - ew) ? (p < L_old ? stage[off + p] : y[kHalo + p - L_old]) : 0;
                w += dw;
                i += di;
                if (i >= a.D) {
                    i -= a.D;
                    ++w;
                }
            }
            fence_proxy_async();  // the bulk copy below reads the message through the async proxy
            __syncwarp();
        }
    }

    // ---- probe share (unless finished before the wait) ----
    if (warp >= 1) {
        if (late) {  // the partial sums only now: this launch waits for the first-layer kernel here
            pdl_wait();
            mlp_finish(u0m + tid - kWarp);
        } else if (mlp) {
            // finished after the verification (mlp_early)
        } else if (gather) {
            zp = dot8_bf16(gw, gh, 0.f);  // zero words for a thread past the slice
            for (int v = v0 + tid - kWarp + (kRescanThreads - kWarp); v < v1; v += kRescanThreads - kWarp)
                zp = dot8_bf16(__ldg(w4 + v), __ldg(h4 + v), zp);
        } else if (!pf_probe) {
            probe_dot(h4);
        }
    }
    if (!probe_ok) key = kKeyTimeout;
    const float z_w = warp_sum_f32(zp);

    // ---- the continuation of this warp's best match: lane j (1..kw) gathers tokens 4(j-1) .. +3 ----
    uint4 cw = make_uint4(0, 0, 0, 0);
    if (key != 0u && key != kKeyTimeout && lane >= 1 && lane <= kw) {
        const int32_t e = int32_t(key & kKeyEndMask);
        const int32_t len = min(a.k, L - 1 - e);
        int32_t t4[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int32_t i = 4 * (lane - 1) + q;
            const int32_t p = e + 1 + i;
            t4[q] = i < len ? (p < L_old ? stage[off + p] : y[kHalo + p - L_old]) : 0;
        }
        cw = make_uint4(uint32_t(t4[0]), uint32_t(t4[1]), uint32_t(t4[2]), uint32_t(t4[3]));
    }

    // ---- ship to the leader ----
    cluster_wait_acquire();  // every CTA has read the length and the leader's barrier is initialised
    const uint32_t done_addr = map_to_rank(&bars[3], lead);
    unsigned char *slot = msgs + size_t(rank * kRescanWarps + warp) * slot_bytes;
    if (lane == 0) {
        uint4 h;
        h.x = key;
        h.y = __float_as_uint(z_w);
        h.z = 0u;
        h.w = 0u;
        st_async_v4(map_to_rank(slot, lead), h, done_addr);
    } else if (lane <= kw) {
        st_async_v4(map_to_rank(slot + 16 * lane, lead), cw, done_addr);
    }
    if (kCand && warp == 0 && lane == 0)  // this CTA's candidates, in one bulk copy
        bulk_s2c(map_to_rank(cmsgs + size_t(rank) * cl.cslot, lead), cstage, cl.cslot, done_addr);
    if (rank != lead || warp != 0) {
        if (kCand && warp == 0 && lane == 0) bulk_wait_read();  // the message has been read out
        if (timed_out && lane == 0) {  // copies still in flight get a second bounded wait
            (void)mbar_wait(&bars[0], 0);
            (void)mbar_wait(&bars[1], 0);
        }
        if (!probe_ok && lane == 0) (void)mbar_wait(&bars[2], 0);
        return;
    }

    // ---- leader, warp 0: the append, then the row's answer ----
    if (verifying) {
        for (int32_t i = lane; i <= acc; i += kWarp) row[L_old + i] = y[kHalo + i];
        if (lane == 0 && len_ok) {
            a.lens[b] = L;
            a.out_accept[b] = acc;
        }
    }
    const bool all_in = __all_sync(kFull, mbar_wait_polls(&bars[3], 0, a.msg_wait_polls));
    uint32_t k_r = 0u;
    int32_t i_r = 0;
    float z_r = 0.f;
    if (all_in) {
        for (int i = lane; i < nmsg; i += kWarp) {  // lane j: messages j, j + 32, ... in order
            const uint2 hv = *reinterpret_cast<const uint2 *>(msgs + size_t(i) * slot_bytes);
            z_r += __uint_as_float(hv.y);
            if (hv.x > k_r) {
                k_r = hv.x;
                i_r = i;
            }
        }
    }
    const uint32_t best = all_in ? __reduce_max_sync(kFull, k_r) : kKeyTimeout;
    const unsigned at = __ballot_sync(kFull, k_r == best);
    const int32_t win = __shfl_sync(kFull, i_r, at != 0u ? __ffs(at) - 1 : 0);
    const float z = warp_sum_f32(z_r) + (mlp ? a.b2 : 0.f);
    const bool timeout = best == kKeyTimeout;
    const bool hit = len_ok && !timeout && best != 0u;
    const int32_t n = hit ? int32_t(best >> kKeyShift) : 0;
    const int32_t e = hit ? int32_t(best & kKeyEndMask) : -1;
    const int32_t kappa = a.kappa > 0 ? a.kappa : a.n_min;
    if constexpr (kCand) {
        // The row's candidates, most recent first: the appended ends (highest first), then the CTAs' lists
        // from the leader's (the most recent range) down to CTA 0's.  s_sel[w] is merged candidate w's
        // source: -1 - j for the appended end L_old - 1 + j, else r kMaxCand + i for entry i of CTA r.
        auto count_of = [&](int r) {
            return min(*reinterpret_cast<const int32_t *>(cmsgs + size_t(r) * cl.cslot), a.W);
        };
        const int n_new = hit ? __popc(new_c[0]) + __popc(new_c[1]) + __popc(new_c[2]) : 0;
        int total = n_new;
        if (hit)
            for (int r = 0; r < int(C); ++r) total += count_of(r);
        const int ncand = min(total, a.W);
        int32_t mode = SWITCHSD_MODE_NO_REP;
        if (hit) mode = (ncand > 0 && z >= a.logit_tau) ? SWITCHSD_MODE_COPY : SWITCHSD_MODE_REP_NO_COPY;
        const int nc = mode == SWITCHSD_MODE_COPY ? ncand : 0;
        if (lane < nc) {
            int src = 0;
            if (lane < n_new) {
                int k = lane, j = -1;
                for (int t = 2; t >= 0 && j < 0; --t) {
                    const int pc = __popc(new_c[t]);
                    if (k < pc) {
                        uint32_t mm = new_c[t];
                        for (int q = 0; q < k; ++q) mm &= ~(1u << (31 - __clz(mm)));
                        j = 32 * t + 31 - __clz(mm);
                    } else {
                        k -= pc;
                    }
                }
                src = -1 - j;
            } else {
                int k = lane - n_new, r = int(C) - 1;
                for (; r > 0; --r) {
                    const int cr = count_of(r);
                    if (k < cr) break;
                    k -= cr;
                }
                src = r * kMaxCand + k;
            }
            s_sel[lane] = src;
        }
        __syncwarp();
        const int cwE = (a.W + 3) / 4;
        auto cand_end = [&](int src) -> int32_t {
            if (src < 0) return L_old - 2 - src;  // L_old - 1 + j with j = -1 - src
            const int r = src / kMaxCand;
            return reinterpret_cast<const int32_t *>(cmsgs + size_t(r) * cl.cslot + 16)[src - r * kMaxCand];
        };
        if (lane < nc) a.out_cand_len[size_t(b) * a.W + lane] = min(a.D, L - 1 - cand_end(s_sel[lane]));
        const int dw = kWarp / a.D, di = kWarp - dw * a.D;  // (candidate, token) step of 32 slots
        int w = lane / a.D, i = lane - w * a.D;
        for (int t = lane; t < nc * a.D; t += kWarp, w += dw, i += di) {
            if (i >= a.D) {
                i -= a.D;
                ++w;
            }
            const int src = s_sel[w];
            const int32_t ew = cand_end(src);
            if (i < min(a.D, L - 1 - ew)) {
                int32_t tok;
                if (src < 0) {
                    tok = y[kHalo + ew + 1 + i - L_old];
                } else {
                    const int r = src / kMaxCand;
                    tok = reinterpret_cast<const int32_t *>(cmsgs + size_t(r) * cl.cslot + 16 + 16 * cwE)
                        [(src - r * kMaxCand) * a.D + i];
                }
                a.out_cand[(size_t(b) * a.W + w) * a.D + i] = tok;
            }
        }
        if (lane == 0) {
            a.out_mode[b] = mode;
            a.out_score[b] = z;
            a.out_ncand[b] = nc;
            if (a.out_match_n) a.out_match_n[b] = n;
            if (a.out_match_end) a.out_match_end[b] = e;
            if (verifying && !len_ok) a.out_accept[b] = -1;
            if (verifying && a.out_choice) a.out_choice[b] = len_ok ? choice : 0;
            if (a.status) {
                int32_t st = vst;
                if (st == SWITCHSD_ROW_OK && timeout) st = SWITCHSD_ROW_TIMEOUT;
                a.status[b] = st;
            }
            bulk_wait_read();  // the leader's own message has been read out
        }
        (void)win;
    } else {
        const int32_t kappa = a.kappa > 0 ? a.kappa : a.n_min;
        int32_t mode = SWITCHSD_MODE_NO_REP;
        if (hit) mode = (n >= kappa && z >= a.logit_tau) ? SWITCHSD_MODE_COPY : SWITCHSD_MODE_REP_NO_COPY;
        const int32_t len = mode == SWITCHSD_MODE_COPY ? min(a.k, L - 1 - e) : 0;
        if (lane == 0) {
            if (a.counters) count_row(a.counters, mode, verifying, a.out_mode[b], acc);  // out_mode: the previous mode
            a.out_mode[b] = mode;
            a.out_len[b] = len;
            a.out_score[b] = z;
            if (a.out_match_n) a.out_match_n[b] = n;
            if (a.out_match_end) a.out_match_end[b] = e;
            if (verifying && !len_ok) a.out_accept[b] = -1;
            if (a.status) {
                int32_t st = vst;
                if (st == SWITCHSD_ROW_OK && timeout) st = SWITCHSD_ROW_TIMEOUT;
                a.status[b] = st;
            }
        }
        const int32_t *wd = reinterpret_cast<const int32_t *>(msgs + size_t(win) * slot_bytes + 16);
        for (int i = lane; i < len; i += kWarp) a.out_draft[size_t(b) * a.k + i] = wd[i];
    }
    if (!all_in && lane == 0) (void)mbar_wait(&bars[3], 0);  // messages still in flight: a second bounded wait
    if (timed_out && lane == 0) {
        (void)mbar_wait(&bars[0], 0);
        (void)mbar_wait(&bars[1], 0);
    }
    if (!probe_ok && lane == 0) (void)mbar_wait(&bars[2], 0);
}

size_t rescan_smem_bytes(const StepArgs &args, int split) {
    const bool cand = args.W > 0;
    const size_t stage = size_t((kHalo + args.tile + kFwd + 3) & ~3) * sizeof(int32_t);
    const size_t probe = 2 * size_t(args.probe_words) * 16 + size_t(args.hash_words) * 4;
    const size_t msgs = size_t(split) * kRescanWarps * 16 * size_t(1 + (cand ? 0 : ((args.k + 3) >> 2)));
    if (!cand) return stage + probe + msgs;
    const CandLayout c = cand_layout(args.tile, args.W, args.D);
    return stage + probe + msgs + size_t(split + 1) * c.cslot + size_t(c.bm_words + c.v_ints) * sizeof(int32_t);
}

template <bool kSampled, bool kCand, bool kPre, bool kMlp>
static cudaError_t rescan_attrs() {
    static bool attr_done[64] = {false};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && !attr_done[dev]) {
        cudaError_t e = cudaFuncSetAttribute(rescan_kernel<kSampled, kCand, kPre, kMlp>,
                                             cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        if (e != cudaSuccess) return e;
        e = cudaFuncSetAttribute(rescan_kernel<kSampled, kCand, kPre, kMlp>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 int(kRescanSmemBudget));
        if (e != cudaSuccess) return e;
        attr_done[dev] = true;
    }
    return cudaSuccess;
}

template <bool kSampled, bool kCand, bool kPre, bool kMlp>
static cudaError_t launch_rescan(const StepArgs &args, int split, cudaStream_t stream) {
    const cudaError_t e = rescan_attrs<kSampled, kCand, kPre, kMlp>();
    if (e != cudaSuccess) return e;
    return launch_pdl(rescan_kernel<kSampled, kCand, kPre, kMlp>, dim3(unsigned(split), unsigned(args.B), 1),
                      dim3(kRescanThreads, 1, 1), rescan_smem_bytes(args, split), stream, unsigned(split), args);
}

// Resident CTAs per SM of an instance at a dynamic shared-memory size (cached: the occupancy calculator
// runs once per instance, device and size).
template <bool kSampled, bool kCand, bool kPre, bool kMlp>
static cudaError_t rescan_per_sm(size_t smem, int &out) {
    struct Entry {
        int dev;
        size_t smem;
        int n;
    };
    static std::mutex mu;
    static Entry cache[32];
    static int used = 0;
    int dev = 0;
    cudaGetDevice(&dev);
    {
        std::lock_guard<std::mutex> lk(mu);
        for (int i = 0; i < used; ++i)
            if (cache[i].dev == dev && cache[i].smem == smem) {
                out = cache[i].n;
                return cudaSuccess;
            }
    }
    cudaError_t e = rescan_attrs<kSampled, kCand, kPre, kMlp>();
    if (e != cudaSuccess) return e;
    int n = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, rescan_kernel<kSampled, kCand, kPre, kMlp>, kRescanThreads, smem);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lk(mu);
    if (used < 32) cache[used++] = Entry{dev, smem, n};
    out = n;
    return cudaSuccess;
}

template <bool kSampled, bool kCand, bool kMlp>
static cudaError_t choose_hash(StepArgs &args, int split, int sms) {
    const int32_t words = int32_t(((args.tile + 3) / 4 + 3) & ~3);  // one byte an end; 16-byte multiple
    args.hash_words = 0;
    // The hashing overlaps the preceding launch only when this launch's CTAs are resident early, which a
    // grid of fewer CTAs than SMs is not, measured: the 8K rows (two CTAs a row, 128 CTAs) lose 0.1 us a
    // launch with it, the 32K rows (512 CTAs) gain 0.1 us and the 128K rows (256 CTAs of 8.5K ends) 0.8 us.
    if (int64_t(split) * args.B < int64_t(sms)) return cudaSuccess;
    int without = 0, with = 0;
    cudaError_t e = rescan_per_sm<kSampled, kCand, false, kMlp>(rescan_smem_bytes(args, split), without);
    if (e != cudaSuccess) return e;
    StepArgs h = args;
    h.hash_words = words;
    const size_t bytes = rescan_smem_bytes(h, split);
    if (bytes > kRescanSmemBudget) return cudaSuccess;
    e = rescan_per_sm<kSampled, kCand, true, kMlp>(bytes, with);
    if (e != cudaSuccess) return e;
    if (with >= 1 && with >= (without < kRescanMinBlocks ? without : kRescanMinBlocks)) args.hash_words = words;
    return cudaSuccess;
}

template <bool kSampled, bool kCand>
static cudaError_t choose_hash2(StepArgs &args, int split, int sms) {
    return args.z1_part != nullptr ? choose_hash<kSampled, kCand, true>(args, split, sms)
                                   : choose_hash<kSampled, kCand, false>(args, split, sms);
}

cudaError_t rescan_choose_hash(StepArgs &args, int split, int sms) {
    if (args.W > 0) return choose_hash2<false, true>(args, split, sms);
    return args.pv_p != nullptr ? choose_hash2<true, false>(args, split, sms)
                                : choose_hash2<false, false>(args, split, sms);
}

template <bool kSampled, bool kCand>
static cudaError_t launch_rescan2(const StepArgs &args, int split, cudaStream_t stream) {
    const bool mlp = args.z1_part != nullptr;
    if (args.hash_words > 0)
        return mlp ? launch_rescan<kSampled, kCand, true, true>(args, split, stream)
                   : launch_rescan<kSampled, kCand, true, false>(args, split, stream);
    return mlp ? launch_rescan<kSampled, kCand, false, true>(args, split, stream)
               : launch_rescan<kSampled, kCand, false, false>(args, split, stream);
}

cudaError_t launch_rescan_kernel(const StepArgs &args, int split, cudaStream_t stream) {
    // candidate verification is greedy (the candidates' targets are compared token by token)
    if (args.W > 0) return launch_rescan2<false, true>(args, split, stream);
    return args.pv_p != nullptr ? launch_rescan2<true, false>(args, split, stream)
                                : launch_rescan2<false, false>(args, split, stream);
}

}  // namespace switchsd
