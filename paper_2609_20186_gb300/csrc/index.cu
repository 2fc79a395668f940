// index.cu -- incremental n-gram index: the same (n*, e*) as the rescan, from hash chains.
//
// For every row b and every n in [n_min, n_max] the index keeps
//   heads[n][b][bucket]  the most recent end position e whose n-gram x[e-n+1..e] hashes to bucket,
//   prev[n][b][e]        the previous end position with the same bucket (-1 at the end of a chain).
// Contexts only grow and positions are inserted in increasing order, so every chain lists end
// positions in decreasing order.  Looking up the suffix n-gram walks its bucket's chain from the head,
// skips the suffix's own end (L-1) and compares candidates token by token; the first exact match is
// the most recent earlier occurrence (§3.3's recency ranking).  n* is the largest n with a match and
// e* its end: exactly the rescan's answer, hash collisions included (they only lengthen the walk).
//
// index_kernel runs one CTA per row with one warp per n and does, in order:
//   verification of the previous draft (as switchsd_verify) and its append, when verifying;
//   insertion of the appended end positions (all lanes at once; positions of one run that fall into
//   the same bucket are linked through __match_any_sync, so one read of the old heads suffices);
//   the lookup, the probe and the switch / copy draft (as switchsd_step), when stepping.
// Candidate mode (W > 0, as switchsd_step_candidates / switchsd_verify_candidates): the previous W
// candidates are verified and the longest accepted one appended; the warp of n = kappa walks its
// chain on past the first match and lists the W most recent ends whose kappa-gram equals the
// suffix's -- exactly the ends whose common suffix with the current one reaches kappa.
#include <new>

#include "common.cuh"
#include "index.cuh"
#include "mlp.cuh"

struct switchsd_index {
    int32_t B, cap, n_min, n_max, nn, log2_buckets;
    int32_t *heads;  // [nn][B][1 << log2_buckets]
    int32_t *prev;   // [nn][B][cap]
    int device;
};

namespace switchsd {

constexpr int kIdxMaxWarps = SWITCHSD_NMAX;
constexpr int kIdxTail = SWITCHSD_NMAX + SWITCHSD_KMAX + 1;  // staged context tail: old end +- the append

// Multiply-xorshift hash of the n tokens ending at the last one (`tok(i)` = token i steps back).
template <typename Tok>
__device__ __forceinline__ uint32_t gram_hash(int n, Tok tok, int log2_buckets) {
    uint64_t h = 0x243F6A8885A308D3ull ^ uint64_t(n);
    for (int i = 0; i < n; ++i) {
        h = (h ^ uint64_t(uint32_t(tok(i)))) * 0x9E3779B97F4A7C15ull;
        h ^= h >> 29;
    }
    return uint32_t(h >> (64 - log2_buckets));
}

struct IndexArgs {
    int32_t *ctx, *lens;
    const uint16_t *hidden, *probe_w;
    const float *z1_part;  // two-layer probe: split-K partial sums of W1 h [mlp_S][B][H1p], else null
    const float *b1;       // two-layer probe: first-layer biases (null = zero) and output weights
    const uint16_t *w2;
    int32_t mlp_S, H1, H1p;
    float b2;
    const int32_t *pv_draft, *pv_target, *pv_len;  // verification inputs (null: no verification)
    const float *pv_p, *pv_q, *pv_u;               // sampled verification (null p: greedy)
    int32_t hidden_rows;                           // > 1: the probe reads row a_b of [B, hidden_rows, d]
    int32_t *out_accept;
    int32_t *out_draft, *out_len, *out_mode;
    float *out_score;
    int32_t *out_match_n, *out_match_end, *status;
    int32_t *heads, *prev;
    int32_t B, cap, d, k, n_min, n_max, kappa, log2_buckets, stepping;
    float logit_tau;
    // candidate mode (W > 0): W candidates of up to D tokens; pv_draft / pv_target / pv_len then hold
    // the previous candidates [B][W][D], their targets [B][W][D+1] and counts [B]
    int32_t W, D;
    const int32_t *pv_cand_len;  // [B][W]
    int32_t *out_choice, *out_cand, *out_cand_len, *out_ncand;
    int32_t prefetch;  // SWITCHSD_PREFETCH_* bits: the inputs they name are read before the wait
    unsigned long long *counters;  // optional per-mode tallies (switchsd_params.counters), else null
};

// This thread's share of the linear probe's dot product over row b's hidden state (threads stride the
// d/8 words; the same partition wherever it is computed, so the logit is the same).
__device__ __forceinline__ float index_probe_partial(const IndexArgs &a, int b, int32_t hrow) {
    const uint4 *h4 = reinterpret_cast<const uint4 *>(
        a.hidden + (size_t(b) * size_t(a.hidden_rows > 1 ? a.hidden_rows : 1) + size_t(hrow)) * a.d);
    const uint4 *w4 = reinterpret_cast<const uint4 *>(a.probe_w);
    float zp = 0.f;
    for (int v = threadIdx.x; v < (a.d >> 3); v += blockDim.x) {
        const uint4 w = __ldg(w4 + v), h = __ldg(h4 + v);
        zp = fmaf(bf16_lo(w.x), bf16_lo(h.x), zp);
        zp = fmaf(bf16_hi(w.x), bf16_hi(h.x), zp);
        zp = fmaf(bf16_lo(w.y), bf16_lo(h.y), zp);
        zp = fmaf(bf16_hi(w.y), bf16_hi(h.y), zp);
        zp = fmaf(bf16_lo(w.z), bf16_lo(h.z), zp);
        zp = fmaf(bf16_hi(w.z), bf16_hi(h.z), zp);
        zp = fmaf(bf16_lo(w.w), bf16_lo(h.w), zp);
        zp = fmaf(bf16_hi(w.w), bf16_hi(h.w), zp);
    }
    return zp;
}

__global__ void __launch_bounds__(kIdxMaxWarps * kWarp) index_kernel(const IndexArgs a) {
    __shared__ int32_t s_tail[kIdxTail];     // x[L_old - NMAX .. L_old + KMAX]
    __shared__ int32_t s_ver[3];             // accepted, new length, status
    __shared__ int32_t s_found[kIdxMaxWarps];
    __shared__ float s_wz[kIdxMaxWarps];
    __shared__ int32_t s_out[3];
    __shared__ int32_t s_cend[SWITCHSD_WMAX];  // candidate mode: the listed ends, most recent first
    __shared__ int32_t s_ncf;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int nwarps = blockDim.x >> 5;
    const int b = blockIdx.x;
    const bool verifying = a.pv_len != nullptr;
    // With the prefetch bits (the caller's promise that the preceding kernel writes neither) the row's
    // length and tail, and the linear probe of row 0 of its state, are read before the wait.
    const bool pf_ctx = (a.prefetch & SWITCHSD_PREFETCH_CONTEXT) != 0;
    const bool pf_probe = (a.prefetch & SWITCHSD_PREFETCH_PROBE) != 0 && a.stepping && a.z1_part == nullptr &&
                          a.hidden_rows <= 1;
    float zp_early = 0.f;
    if (pf_probe) zp_early = index_probe_partial(a, b, 0);
    if (!pf_ctx) pdl_wait();

    if (tid == 0) s_ncf = 0;
    int32_t *row = a.ctx + size_t(b) * a.cap;
    const int32_t L_old = a.lens[b];
    const bool len_ok = L_old >= 1 && L_old <= a.cap;
    const int32_t tail0 = L_old - SWITCHSD_NMAX;  // s_tail[i] = x[tail0 + i]
    for (int i = tid; i < SWITCHSD_NMAX; i += blockDim.x) {
        const int32_t p = tail0 + i;
        s_tail[i] = (len_ok && p >= 0) ? row[p] : 0;
    }
    if (pf_ctx) pdl_wait();  // the previous draft, the target and the index tables come after this
    pdl_trigger();
    if (warp == 0) {
        int32_t acc = -1, L = L_old, vst = len_ok ? SWITCHSD_ROW_OK : SWITCHSD_ROW_BAD_LEN;
        int32_t choice = 0;
        if (verifying && len_ok && a.W > 0) {
            // The previous W candidates: lane i tests positions i and i + 32 of each; the longest
            // accepted one is kept (the lowest index on a tie).  ncand = 0 is one empty candidate.
            const int32_t nc = a.pv_len[b];
            bool badlen = nc < 0 || nc > a.W;
            const int ncx = badlen ? 0 : (nc > 0 ? nc : 1);
            int32_t best = -1;
            for (int w = 0; w < ncx; ++w) {
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
                    choice = w;
                }
            }
            if (badlen) {
                vst = SWITCHSD_ROW_BAD_LEN;
                choice = 0;
            } else if (L_old + best + 1 > a.cap) {
                vst = SWITCHSD_ROW_CAPACITY;
            } else {
                const size_t o = size_t(b) * a.W + choice;
                const int32_t *c = a.pv_draft + o * a.D;
                const int32_t tb = a.pv_target[o * (a.D + 1) + best];
                for (int i = lane; i <= best; i += kWarp) {
                    const int32_t t = i < best ? c[i] : tb;
                    s_tail[SWITCHSD_NMAX + i] = t;
                    row[L_old + i] = t;
                }
                acc = best;
                L = L_old + best + 1;
            }
        } else if (verifying && len_ok) {
            const int32_t n = a.pv_len[b];
            if (n < 0 || n > a.k) {
                vst = SWITCHSD_ROW_BAD_LEN;
            } else {
                const int32_t *dr = a.pv_draft + size_t(b) * a.k;
                const int32_t *tg = a.pv_target + size_t(b) * (a.k + 1);
                acc = n;
                for (int base = 0; base < n; base += kWarp) {
                    const int i = base + lane;
                    // greedy: a draft token is rejected when it differs from the target's; sampled: when
                    // u * q (binary32) is not below p
                    bool rej = false;
                    if (i < n) {
                        if (a.pv_p != nullptr) {
                            const size_t o = size_t(b) * a.k + i;
                            rej = !(__fmul_rn(a.pv_u[o], a.pv_q ? a.pv_q[o] : 1.f) < a.pv_p[o]);
                        } else {
                            rej = dr[i] != tg[i];
                        }
                    }
                    const unsigned m = __ballot_sync(kFull, rej);
                    if (m) {
                        acc = base + __ffs(m) - 1;
                        break;
                    }
                }
                if (L_old + acc + 1 > a.cap) {
                    vst = SWITCHSD_ROW_CAPACITY;
                    acc = -1;
                } else {
                    for (int i = lane; i <= acc; i += kWarp) {
                        const int32_t t = i < acc ? dr[i] : tg[acc];
                        s_tail[SWITCHSD_NMAX + i] = t;
                        row[L_old + i] = t;
                    }
                    L = L_old + acc + 1;
                }
            }
        }
        if (lane == 0) {
            s_ver[0] = acc;
            s_ver[1] = L;
            s_ver[2] = vst;
            if (verifying && len_ok) {
                a.lens[b] = L;
                a.out_accept[b] = acc;
            } else if (verifying) {
                a.out_accept[b] = -1;
            }
            if (verifying && a.W > 0 && a.out_choice) a.out_choice[b] = choice;
            if (!a.stepping && a.status) a.status[b] = vst;
        }
    }
    __syncthreads();
    const int32_t L = s_ver[1];
    const int n = a.n_min + warp;  // this warp's gram length
    const bool has_n = warp < a.n_max - a.n_min + 1;
    const size_t nb = size_t(1) << a.log2_buckets;
    int32_t *heads = a.heads + (size_t(warp) * a.B + b) * nb;
    int32_t *prev = a.prev + (size_t(warp) * a.B + b) * a.cap;
    auto tail_tok = [&](int32_t p) { return s_tail[p - tail0]; };  // valid for p in [tail0, L)

    // Insert the appended end positions p in [L_old, L) (lanes over p, chained through match_any).
    if (has_n && L > L_old) {
        for (int32_t base = L_old; base < L; base += kWarp) {
            const int32_t p = base + lane;
            const bool valid = p < L && p >= n - 1;
            uint32_t bucket = 0xffffffffu;
            if (valid) bucket = gram_hash(n, [&](int i) { return tail_tok(p - i); }, a.log2_buckets);
            const unsigned peers = __match_any_sync(kFull, bucket) & __ballot_sync(kFull, valid);
            const int32_t old_head = valid ? heads[bucket] : -1;
            __syncwarp();  // every lane has read its head before any lane replaces one
            // A head at or past p means these positions were inserted before (the same tokens appended
            // again after the lengths were rewound): the chains already hold them, so leave them be.
            // This keeps prev[p] < p, so every chain stays acyclic.
            if (valid && old_head < p) {
                const unsigned earlier = peers & ((1u << lane) - 1u);
                prev[p] = earlier ? base + (31 - __clz(earlier)) : old_head;
                if ((peers >> lane) == 1u) heads[bucket] = p;  // the latest position of the run
            }
            __syncwarp();
        }
    }
    if (!a.stepping) return;

    // Lookup: the most recent earlier occurrence of the suffix n-gram, if any.  Candidate mode: the
    // warp of n = kappa lists the W most recent.
    const int32_t kappa_c = a.kappa > 0 ? a.kappa : a.n_min;
    const bool collect = a.W > 0 && has_n && n == kappa_c;
    int32_t found = -1, nfound = 0;
    if (has_n && len_ok && L >= n + 1) {
        const uint32_t bucket = gram_hash(n, [&](int i) { return tail_tok(L - 1 - i); }, a.log2_buckets);
        const int32_t mine = lane < n ? tail_tok(L - 1 - lane) : 0;
        int32_t e = heads[bucket];
        // A valid chain strictly decreases and ends at -1 within L hops; the bounds keep a stale or
        // unbuilt index from reading outside its tables.
        for (int32_t hops = 0; e >= 0 && e < a.cap && hops < a.cap; ++hops) {
            if (e <= L - 2 && e >= n - 1) {
                const bool eq = lane >= n || (e - lane >= L_old ? tail_tok(e - lane) : row[e - lane]) == mine;
                if (__all_sync(kFull, eq)) {
                    if (found < 0) found = e;
                    if (!collect) break;
                    if (lane == 0) s_cend[nfound] = e;
                    if (++nfound >= a.W) break;
                }
            }
            e = prev[e];
        }
    }
    if (lane == 0 && warp < kIdxMaxWarps) s_found[warp] = found;
    if (collect && lane == 0) s_ncf = nfound;

    // Probe partial over the whole hidden vector (linear probe), or over every unit of the two-layer
    // probe: the S split-K partial sums in order, then b1, ReLU and w2.
    float zp = 0.f;
    if (a.z1_part != nullptr) {
        for (int u = tid; u < a.H1; u += blockDim.x) {
            float z1 = 0.f;
            for (int s = 0; s < a.mlp_S; ++s) z1 += a.z1_part[(size_t(s) * a.B + size_t(b)) * a.H1p + u];
            const float bias = a.b1 ? a.b1[u] : 0.f;
            zp = fmaf(bf16_lo(uint32_t(a.w2[u])), fmaxf(z1 + bias, 0.f), zp);
        }
    } else if (pf_probe) {
        zp = zp_early;
    } else {
        const int32_t hrow = a.hidden_rows > 1 && s_ver[0] > 0 ? s_ver[0] : 0;  // row a_b when gathering
        zp = index_probe_partial(a, b, hrow);
    }
    zp = warp_sum_f32(zp);
    if (lane == 0) s_wz[warp] = zp;
    __syncthreads();

    if (tid == 0) {
        float z = 0.f;
        for (int w = 0; w < nwarps; ++w) z += s_wz[w];
        if (a.z1_part != nullptr) z += a.b2;
        int32_t nstar = 0, estar = -1;
        for (int w = a.n_max - a.n_min; w >= 0; --w)
            if (s_found[w] >= 0) {
                nstar = a.n_min + w;
                estar = s_found[w];
                break;
            }
        const bool hit = len_ok && nstar > 0;
        const bool gate = a.W > 0 ? s_ncf > 0 : nstar >= kappa_c;
        int32_t mode = SWITCHSD_MODE_NO_REP;
        if (hit) mode = (gate && z >= a.logit_tau) ? SWITCHSD_MODE_COPY : SWITCHSD_MODE_REP_NO_COPY;
        const int32_t len = (a.W == 0 && mode == SWITCHSD_MODE_COPY) ? min(a.k, L - 1 - estar) : 0;
        s_out[0] = estar;
        s_out[1] = len;
        s_out[2] = mode == SWITCHSD_MODE_COPY ? s_ncf : 0;  // candidate mode: candidates written
        if (a.W == 0 && a.counters)  // out_mode still holds the previous step's mode
            count_row(a.counters, mode, verifying, a.out_mode[b], s_ver[0]);
        a.out_mode[b] = mode;
        if (a.W == 0) a.out_len[b] = len;
        else a.out_ncand[b] = s_out[2];
        a.out_score[b] = z;
        if (a.out_match_n) a.out_match_n[b] = nstar;
        if (a.out_match_end) a.out_match_end[b] = estar;
        if (a.status) a.status[b] = s_ver[2];
    }
    __syncthreads();
    if (a.W > 0) {
        // The candidates' continuations x[e_w+1 .. e_w+len_w], len_w = min(D, L-1-e_w).
        const int32_t nc = s_out[2];
        for (int t = tid; t < nc * a.D; t += blockDim.x) {
            const int w = t / a.D, i = t - w * a.D;
            const int32_t ew = s_cend[w];
            const int32_t lw = min(a.D, L - 1 - ew);
            const int32_t p = ew + 1 + i;
            if (i == 0) a.out_cand_len[size_t(b) * a.W + w] = lw;
            if (i < lw) a.out_cand[(size_t(b) * a.W + w) * a.D + i] = p >= L_old ? tail_tok(p) : row[p];
        }
        return;
    }
    const int32_t e = s_out[0], len = s_out[1];
    // The copy draft x[e+1 .. e+len]: positions below L_old are in global memory, the rest in s_tail.
    for (int i = tid; i < len; i += blockDim.x) {
        const int32_t p = e + 1 + i;
        a.out_draft[size_t(b) * a.k + i] = p >= L_old ? tail_tok(p) : row[p];
    }
}

// Build: positions n-1 .. L-1 of every (row, n) inserted in increasing order, 32 per warp iteration.
__global__ void __launch_bounds__(256) index_build_kernel(const int32_t *ctx, const int32_t *lens, int32_t *heads_all,
                                                          int32_t *prev_all, int32_t B, int32_t cap, int32_t n_min,
                                                          int32_t nn, int32_t log2_buckets) {
    const int lane = threadIdx.x & 31;
    const int gw = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;  // one warp per (n, row)
    pdl_wait();
    pdl_trigger();
    if (gw >= nn * B) return;
    const int w = gw / B, b = gw % B;
    const int n = n_min + w;
    const size_t nb = size_t(1) << log2_buckets;
    int32_t *heads = heads_all + (size_t(w) * B + b) * nb;
    int32_t *prev = prev_all + (size_t(w) * B + b) * cap;
    const int32_t *row = ctx + size_t(b) * cap;
    int32_t L = lens[b];
    if (L < 0 || L > cap) L = 0;
    for (int32_t base = 0; base < L; base += kWarp) {
        const int32_t p = base + lane;
        const bool valid = p < L && p >= n - 1;
        uint32_t bucket = 0xffffffffu;
        if (valid) bucket = gram_hash(n, [&](int i) { return row[p - i]; }, log2_buckets);
        const unsigned peers = __match_any_sync(kFull, bucket) & __ballot_sync(kFull, valid);
        const int32_t old_head = valid ? heads[bucket] : -1;
        __syncwarp();  // every lane has read its head before any lane replaces one
        if (valid) {
            const unsigned earlier = peers & ((1u << lane) - 1u);
            prev[p] = earlier ? base + (31 - __clz(earlier)) : old_head;
            if ((peers >> lane) == 1u) heads[bucket] = p;
        }
        __syncwarp();
    }
}

// ------------------------------------------------------------------------------------------------
// Host side.
// ------------------------------------------------------------------------------------------------
int index_n_min(const switchsd_index *idx) { return idx->n_min; }
int index_n_max(const switchsd_index *idx) { return idx->n_max; }

int index_launch(switchsd_index *idx, int32_t *ctx, int32_t *lens, const uint16_t *hidden, const uint16_t *probe_w,
                 const float *z1_part, const float *b1, const uint16_t *w2, int mlp_S, int H1, int H1p, float b2,
                 const int32_t *pv_draft, const int32_t *pv_target, const int32_t *pv_len, int32_t *out_accept,
                 int32_t *out_draft, int32_t *out_len, int32_t *out_mode, float *out_score, int32_t *out_match_n,
                 int32_t *out_match_end, int32_t *status, int B, int cap, int d, int k, int n_min, int n_max, int kappa,
                 float logit_tau, bool stepping, cudaStream_t stream, const float *pv_p, const float *pv_q,
                 const float *pv_u, int hidden_rows, const IndexCandidates *cand, int prefetch,
                 unsigned long long *counters) {
    if (idx->B != B || idx->cap != cap || idx->n_min != n_min || idx->n_max != n_max) return SWITCHSD_ERR_SHAPE;
    // Candidate mode lists the ends of the kappa-gram chain: kappa must be one of the index's n, or
    // above n_max (no end can then reach it: no candidate, as for the rescan).
    if (cand != nullptr && (kappa > 0 ? kappa : n_min) < n_min) return SWITCHSD_ERR_SHAPE;
    IndexArgs a;
    a.W = cand ? cand->W : 0;
    a.D = cand ? cand->D : 0;
    a.pv_cand_len = cand ? cand->pv_cand_len : nullptr;
    a.out_choice = cand ? cand->out_choice : nullptr;
    a.out_cand = cand ? cand->out_cand : nullptr;
    a.out_cand_len = cand ? cand->out_cand_len : nullptr;
    a.out_ncand = cand ? cand->out_ncand : nullptr;
    a.prefetch = prefetch;
    a.counters = stepping ? counters : nullptr;
    a.pv_p = pv_p;
    a.pv_q = pv_q;
    a.pv_u = pv_u;
    a.hidden_rows = hidden_rows;
    a.ctx = ctx;
    a.lens = lens;
    a.hidden = hidden;
    a.probe_w = probe_w;
    a.z1_part = z1_part;
    a.b1 = b1;
    a.w2 = w2;
    a.mlp_S = mlp_S;
    a.H1 = H1;
    a.H1p = H1p;
    a.b2 = b2;
    a.pv_draft = pv_draft;
    a.pv_target = pv_target;
    a.pv_len = pv_len;
    a.out_accept = out_accept;
    a.out_draft = out_draft;
    a.out_len = out_len;
    a.out_mode = out_mode;
    a.out_score = out_score;
    a.out_match_n = out_match_n;
    a.out_match_end = out_match_end;
    a.status = status;
    a.heads = idx->heads;
    a.prev = idx->prev;
    a.B = B;
    a.cap = cap;
    a.d = d;
    a.k = k;
    a.n_min = n_min;
    a.n_max = n_max;
    a.kappa = kappa;
    a.log2_buckets = idx->log2_buckets;
    a.stepping = stepping ? 1 : 0;
    a.logit_tau = logit_tau;
    const cudaError_t e = launch_pdl(index_kernel, dim3(unsigned(B)), dim3(unsigned(idx->nn * kWarp)), 0, stream, 0u, a);
    return e == cudaSuccess ? SWITCHSD_OK : SWITCHSD_ERR_CUDA;
}

}  // namespace switchsd

using namespace switchsd;

extern "C" int switchsd_index_create(const switchsd_params *p, switchsd_index **out) {
    if (!p || !out) return SWITCHSD_ERR_ARG;
    *out = nullptr;
    if (p->B < 1 || p->B > 65535 || p->cap < 4 || (p->cap & 3) != 0) return SWITCHSD_ERR_SHAPE;
    if (p->n_min < 1 || p->n_max > SWITCHSD_NMAX || p->n_min > p->n_max) return SWITCHSD_ERR_SHAPE;
    switchsd_index *idx = new (std::nothrow) switchsd_index();
    if (!idx) return SWITCHSD_ERR_CUDA;
    idx->B = p->B;
    idx->cap = p->cap;
    idx->n_min = p->n_min;
    idx->n_max = p->n_max;
    idx->nn = p->n_max - p->n_min + 1;
    int lg = 4;
    while ((int64_t(1) << lg) < 2 * int64_t(p->cap) && lg < 30) ++lg;  // load factor <= 1/2
    idx->log2_buckets = lg;
    cudaGetDevice(&idx->device);
    const size_t heads = size_t(idx->nn) * size_t(p->B) * (size_t(1) << lg) * sizeof(int32_t);
    const size_t prev = size_t(idx->nn) * size_t(p->B) * size_t(p->cap) * sizeof(int32_t);
    if (cudaMalloc(&idx->heads, heads) != cudaSuccess) {
        delete idx;
        return SWITCHSD_ERR_CUDA;
    }
    if (cudaMalloc(&idx->prev, prev) != cudaSuccess) {
        cudaFree(idx->heads);
        delete idx;
        return SWITCHSD_ERR_CUDA;
    }
    *out = idx;
    return SWITCHSD_OK;
}

extern "C" int switchsd_index_build(switchsd_index *idx, const int32_t *ctx_tokens, const int32_t *ctx_lens,
                                    void *stream) {
    if (!idx || !ctx_tokens || !ctx_lens) return SWITCHSD_ERR_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const size_t heads = size_t(idx->nn) * size_t(idx->B) * (size_t(1) << idx->log2_buckets) * sizeof(int32_t);
    if (cudaMemsetAsync(idx->heads, 0xff, heads, s) != cudaSuccess) return SWITCHSD_ERR_CUDA;  // every head = -1
    const int warps = idx->nn * idx->B;
    const cudaError_t e = launch_pdl(index_build_kernel, dim3(unsigned((warps + 7) / 8)), dim3(256), 0, s, 0u,
                                     ctx_tokens, ctx_lens, idx->heads, idx->prev, idx->B, idx->cap, idx->n_min,
                                     idx->nn, idx->log2_buckets);
    return e == cudaSuccess ? SWITCHSD_OK : SWITCHSD_ERR_CUDA;
}

extern "C" size_t switchsd_index_bytes(const switchsd_index *idx) {
    if (!idx) return 0;
    return size_t(idx->nn) * size_t(idx->B) * ((size_t(1) << idx->log2_buckets) + size_t(idx->cap)) * sizeof(int32_t);
}

extern "C" void switchsd_index_destroy(switchsd_index *idx) {
    if (!idx) return;
    int cur = 0;
    cudaGetDevice(&cur);
    if (cur != idx->device) cudaSetDevice(idx->device);
    cudaFree(idx->heads);
    cudaFree(idx->prev);
    if (cur != idx->device) cudaSetDevice(cur);
    delete idx;
}
