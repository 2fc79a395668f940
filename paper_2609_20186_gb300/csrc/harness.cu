// harness.cu -- device stand-in for the neural drafter and the target model (not the controller).
//
// Reads the target's greedy tokens for each row from the caller's future stream and draws the neural
// draft for non-copy rows, with the seeded law stated in switchsd_harness.h.  One warp per row; lane
// i handles draft indices i, i + 32, ...
#include "common.cuh"
#include "switchsd_harness.h"

namespace switchsd {

constexpr int kHarnessThreads = 256;

struct HarnessArgs {
    const int32_t *lens, *mode, *draft, *draft_len, *future;
    int32_t *vdraft, *vlen, *target;  // target: the greedy tokens, or (sampled) the resample tokens
    float *pp, *qq, *uu;              // sampled only
    switchsd_harness_params p;
};

// splitmix64 finaliser (Steele, Lea and Flood; Vigna's published constants).
__device__ __forceinline__ uint64_t splitmix64(uint64_t z) {
    z += 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

__device__ __forceinline__ int32_t token_of(uint64_t r, int32_t V) {
    return int32_t((r >> 32) % uint64_t(V));
}

template <bool kSampled>
__global__ void __launch_bounds__(kHarnessThreads) harness_kernel(const HarnessArgs a) {
    const int lane = threadIdx.x & 31;
    const int b = (blockIdx.x * kHarnessThreads + threadIdx.x) >> 5;
    const switchsd_harness_params &p = a.p;
    pdl_wait();
    pdl_trigger();
    if (b >= p.B) return;
    const int k = p.k;
    const bool copy = a.mode[b] == SWITCHSD_MODE_COPY;
    int len = copy ? a.draft_len[b] : p.gamma;
    len = len < 0 ? 0 : (len > k ? k : len);
    const int32_t L = a.lens[b];
    const uint64_t row_key = splitmix64(splitmix64(splitmix64(p.seed) ^ uint64_t(b)) ^ uint64_t(p.step));
    for (int i = lane; i <= k; i += kWarp) {
        const int64_t pos = int64_t(L) - p.L0 + i;
        const int32_t g = (pos >= 0 && pos < p.n_future) ? a.future[size_t(b) * p.n_future + pos] : 0;
        if (!kSampled) a.target[size_t(b) * (k + 1) + i] = g;
        if (i < k) {
            int32_t d = 0;
            if (i < len) {
                if (copy) {
                    d = a.draft[size_t(b) * k + i];
                } else {
                    const uint64_t slot = 4ull * uint64_t(i);
                    const uint64_t coin = splitmix64(row_key ^ slot) & 0xffffffffull;
                    if (coin < p.thr_neural) {
                        d = g;
                    } else {
                        d = token_of(splitmix64(row_key ^ (slot + 1)), p.V);
                        if (d == g) d = (d + 1) % p.V;
                    }
                }
            }
            a.vdraft[size_t(b) * k + i] = d;
            if (kSampled) {
                const size_t o = size_t(b) * k + i;
                const uint64_t slot = 4ull * uint64_t(i);
                a.pp[o] = i < len ? (d == g ? p.p_hit : p.p_miss) : 0.f;
                a.qq[o] = (i < len && !copy) ? p.q_neural : 1.f;
                a.uu[o] = float(uint32_t(splitmix64(row_key ^ (slot + 2)) >> 40)) * 5.9604644775390625e-8f;  // 2^-24
                int32_t r = 0;
                if (i < len) {
                    r = g;
                    if (g == d) {
                        r = token_of(splitmix64(row_key ^ (slot + 3)), p.V);
                        if (r == d) r = (r + 1) % p.V;
                    }
                }
                a.target[size_t(b) * (k + 1) + i] = r;
            }
        }
        if (kSampled && i >= len) a.target[size_t(b) * (k + 1) + i] = i == len ? g : 0;
    }
    if (lane == 0) a.vlen[b] = len;
}

}  // namespace switchsd

using namespace switchsd;

extern "C" int switchsd_harness_target(const int32_t *ctx_lens, const int32_t *mode, const int32_t *draft,
                                       const int32_t *draft_len, const int32_t *future, int32_t *vdraft,
                                       int32_t *vlen, int32_t *target, const switchsd_harness_params *hp) {
    if (!hp || !ctx_lens || !mode || !draft || !draft_len || !vdraft || !vlen || !target) return SWITCHSD_ERR_ARG;
    if (hp->n_future > 0 && !future) return SWITCHSD_ERR_ARG;
    if (hp->B < 1 || hp->k < 1 || hp->k > SWITCHSD_KMAX || hp->V < 2 || hp->n_future < 0 || hp->gamma < 0 ||
        hp->gamma > hp->k)
        return SWITCHSD_ERR_SHAPE;
    HarnessArgs a;
    a.lens = ctx_lens;
    a.mode = mode;
    a.draft = draft;
    a.draft_len = draft_len;
    a.future = future;
    a.vdraft = vdraft;
    a.vlen = vlen;
    a.target = target;
    a.pp = a.qq = a.uu = nullptr;
    a.p = *hp;
    const int wpb = kHarnessThreads / kWarp;
    const cudaError_t e = launch_pdl(harness_kernel<false>, dim3((hp->B + wpb - 1) / wpb), dim3(kHarnessThreads),
                                     0, static_cast<cudaStream_t>(hp->stream), 0u, a);
    return e == cudaSuccess ? SWITCHSD_OK : SWITCHSD_ERR_CUDA;
}

extern "C" int switchsd_harness_sampled(const int32_t *ctx_lens, const int32_t *mode, const int32_t *draft,
                                        const int32_t *draft_len, const int32_t *future, int32_t *vdraft,
                                        int32_t *vlen, float *p, float *q, float *u, int32_t *resample,
                                        const switchsd_harness_params *hp) {
    if (!hp || !ctx_lens || !mode || !draft || !draft_len || !vdraft || !vlen || !p || !q || !u || !resample)
        return SWITCHSD_ERR_ARG;
    if (hp->n_future > 0 && !future) return SWITCHSD_ERR_ARG;
    if (hp->B < 1 || hp->k < 1 || hp->k > SWITCHSD_KMAX || hp->V < 2 || hp->n_future < 0 || hp->gamma < 0 ||
        hp->gamma > hp->k)
        return SWITCHSD_ERR_SHAPE;
    HarnessArgs a;
    a.lens = ctx_lens;
    a.mode = mode;
    a.draft = draft;
    a.draft_len = draft_len;
    a.future = future;
    a.vdraft = vdraft;
    a.vlen = vlen;
    a.target = resample;
    a.pp = p;
    a.qq = q;
    a.uu = u;
    a.p = *hp;
    const int wpb = kHarnessThreads / kWarp;
    const cudaError_t e = launch_pdl(harness_kernel<true>, dim3((hp->B + wpb - 1) / wpb), dim3(kHarnessThreads),
                                     0, static_cast<cudaStream_t>(hp->stream), 0u, a);
    return e == cudaSuccess ? SWITCHSD_OK : SWITCHSD_ERR_CUDA;
}

// ------------------------------------------------------------------------------------------------
// The stand-in for switchsd_verify_candidates: a copy row's W candidates are verified against the
// target stream (target[w][i] = the stream's token at position L + i for every candidate w: the target's
// greedy token after any prefix the verification can accept); a neural row holds its neural draft as the
// one candidate.  One warp per row.
// ------------------------------------------------------------------------------------------------
namespace switchsd {

struct CandHarnessArgs {
    const int32_t *lens, *mode, *cand, *cand_len, *ncand, *future;
    int32_t *vcand, *vlen, *vn, *target;
    int32_t W, D;
    switchsd_harness_params p;
};

__global__ void __launch_bounds__(kHarnessThreads) harness_candidates_kernel(const CandHarnessArgs a) {
    const int lane = threadIdx.x & 31;
    const int b = (blockIdx.x * kHarnessThreads + threadIdx.x) >> 5;
    const switchsd_harness_params &p = a.p;
    pdl_wait();
    pdl_trigger();
    if (b >= p.B) return;
    const bool copy = a.mode[b] == SWITCHSD_MODE_COPY;
    int n = copy ? a.ncand[b] : 1;
    n = n < 0 ? 0 : (n > a.W ? a.W : n);
    const int gamma = p.gamma < a.D ? p.gamma : a.D;
    const int32_t L = a.lens[b];
    const uint64_t row_key = splitmix64(splitmix64(splitmix64(p.seed) ^ uint64_t(b)) ^ uint64_t(p.step));
    for (int i = lane; i <= a.D; i += kWarp) {
        const int64_t pos = int64_t(L) - p.L0 + i;
        const int32_t g = (pos >= 0 && pos < p.n_future) ? a.future[size_t(b) * p.n_future + pos] : 0;
        for (int w = 0; w < a.W; ++w) {
            const size_t o = size_t(b) * a.W + w;
            a.target[o * (a.D + 1) + i] = w < n ? g : 0;
            if (i < a.D) {
                int32_t d = 0;
                if (w < n) {
                    if (copy) {
                        d = i < a.cand_len[o] ? a.cand[o * a.D + i] : 0;
                    } else if (i < gamma) {
                        const uint64_t slot = 4ull * uint64_t(i);
                        const uint64_t coin = splitmix64(row_key ^ slot) & 0xffffffffull;
                        if (coin < p.thr_neural) {
                            d = g;
                        } else {
                            d = token_of(splitmix64(row_key ^ (slot + 1)), p.V);
                            if (d == g) d = (d + 1) % p.V;
                        }
                    }
                }
                a.vcand[o * a.D + i] = d;
            }
        }
    }
    if (lane < a.W) {
        const size_t o = size_t(b) * a.W + lane;
        a.vlen[o] = lane < n ? (copy ? a.cand_len[o] : gamma) : 0;
    }
    if (lane == 0) a.vn[b] = n;
}

}  // namespace switchsd

extern "C" int switchsd_harness_candidates(const int32_t *ctx_lens, const int32_t *mode, const int32_t *cand,
                                           const int32_t *cand_len, const int32_t *ncand, const int32_t *future,
                                           int32_t W, int32_t D, int32_t *vcand, int32_t *vlen, int32_t *vn,
                                           int32_t *target, const switchsd_harness_params *hp) {
    if (!hp || !ctx_lens || !mode || !cand || !cand_len || !ncand || !vcand || !vlen || !vn || !target)
        return SWITCHSD_ERR_ARG;
    if (hp->n_future > 0 && !future) return SWITCHSD_ERR_ARG;
    if (hp->B < 1 || W < 1 || W > SWITCHSD_WMAX || D < 1 || D > SWITCHSD_KMAX || hp->V < 2 || hp->n_future < 0 ||
        hp->gamma < 0)
        return SWITCHSD_ERR_SHAPE;
    CandHarnessArgs a;
    a.lens = ctx_lens;
    a.mode = mode;
    a.cand = cand;
    a.cand_len = cand_len;
    a.ncand = ncand;
    a.future = future;
    a.vcand = vcand;
    a.vlen = vlen;
    a.vn = vn;
    a.target = target;
    a.W = W;
    a.D = D;
    a.p = *hp;
    const int wpb = kHarnessThreads / kWarp;
    const cudaError_t e = launch_pdl(harness_candidates_kernel, dim3((hp->B + wpb - 1) / wpb), dim3(kHarnessThreads),
                                     0, static_cast<cudaStream_t>(hp->stream), 0u, a);
    return e == cudaSuccess ? SWITCHSD_OK : SWITCHSD_ERR_CUDA;
}

// ------------------------------------------------------------------------------------------------
// switchsd_harness_read: a plain read of what one step reads, the size-matched ceiling for the step
// kernel.  Grid (split, B): CTA (c, b) takes the c-th of `split` equal runs of the 16-byte words that
// hold row b's first ctx_lens[b] tokens, then the c-th run of row b's hidden states, copies them into
// shared memory with bulk (TMA) copies in chunks of up to 64 KB, and xor-folds every word it received
// into out[b * split + c], so no byte is left unread.  prefetch != 0 issues the first chunk's copies
// before the grid-dependency wait (the step kernel's SWITCHSD_PREFETCH_CONTEXT / _PROBE order), else
// after it.  Bulk copies into shared memory read faster than 16-byte loads from every thread on this
// workload's sizes, so this is the faster of the two plain reads.
// ------------------------------------------------------------------------------------------------
namespace switchsd {

constexpr int kReadThreads = 256;
constexpr int32_t kReadChunkWords = 4096;  // 16-byte words per chunk: 64 KB of shared memory

struct ReadArgs {
    const int32_t *ctx, *lens;
    const uint16_t *hidden;
    uint32_t *out;
    int32_t B, cap, d, split, prefetch;
};

__global__ void __launch_bounds__(kReadThreads) read_kernel(const ReadArgs a) {
    extern __shared__ __align__(128) uint4 s_chunk[];
    __shared__ uint64_t s_bar;
    __shared__ uint32_t s_fold[kReadThreads / kWarp];
    const int b = blockIdx.y, c = blockIdx.x;
    if (threadIdx.x == 0) {
        mbar_init(&s_bar, 1);
        fence_mbar_init();
    }
    __syncthreads();
    if (!a.prefetch) pdl_wait();
    int32_t L = a.lens[b];
    L = (L >= 0 && L <= a.cap) ? L : 0;
    const int32_t nw = (L + 3) / 4;  // cap is a multiple of 4: the last word stays inside the row
    const int32_t per = (nw + a.split - 1) / a.split;
    const int32_t w0 = min(nw, c * per), w1 = min(nw, w0 + per);
    const int32_t hw = a.d / 8;
    const int32_t hper = (hw + a.split - 1) / a.split;
    const int32_t h0 = min(hw, c * hper), h1 = min(hw, h0 + hper);
    const uint4 *row = reinterpret_cast<const uint4 *>(a.ctx + size_t(b) * size_t(a.cap)) + w0;
    const uint4 *hrow = reinterpret_cast<const uint4 *>(a.hidden + size_t(b) * size_t(a.d)) + h0;
    // the CTA's words: context [0, nctx) then hidden [nctx, total), in chunks of kReadChunkWords
    const int32_t nctx = w1 - w0, total = nctx + (h1 - h0);
    const int32_t nchunks = (total + kReadChunkWords - 1) / kReadChunkWords;
    auto issue = [&](int32_t i) {  // thread 0: chunk i's copies, completing on s_bar
        const int32_t v0 = i * kReadChunkWords, v1 = min(total, v0 + kReadChunkWords);
        const int32_t c0 = min(v0, nctx), c1 = min(v1, nctx);
        const int32_t g0 = max(v0, nctx) - nctx, g1 = max(v1, nctx) - nctx;
        mbar_arrive_expect_tx(&s_bar, uint32_t(v1 - v0) * 16u);
        if (c1 > c0) bulk_g2s(s_chunk, row + c0, uint32_t(c1 - c0) * 16u, &s_bar);
        if (g1 > g0) bulk_g2s(s_chunk + (c1 - c0), hrow + g0, uint32_t(g1 - g0) * 16u, &s_bar);
    };
    if (threadIdx.x == 0 && nchunks > 0) issue(0);
    if (a.prefetch) pdl_wait();
    pdl_trigger();
    uint32_t acc = 0;
    bool bad = false;
    for (int32_t i = 0; i < nchunks; ++i) {
        const bool arrived = mbar_wait(&s_bar, uint32_t(i & 1));
        if (!__syncthreads_and(arrived)) {  // a copy did not complete in time: leave after waiting once more
            bad = true;
            if (threadIdx.x == 0) mbar_wait(&s_bar, uint32_t(i & 1));
            break;
        }
        const int32_t n = min(total, (i + 1) * kReadChunkWords) - i * kReadChunkWords;
        for (int32_t j = threadIdx.x; j < n; j += kReadThreads) {
            const uint4 v = s_chunk[j];
            acc ^= v.x ^ v.y ^ v.z ^ v.w;
        }
        __syncthreads();  // the buffer is read before the next chunk overwrites it
        if (threadIdx.x == 0 && i + 1 < nchunks) issue(i + 1);
    }
    for (int o = kWarp / 2; o > 0; o >>= 1) acc ^= __shfl_xor_sync(0xffffffffu, acc, o);
    if ((threadIdx.x & (kWarp - 1)) == 0) s_fold[threadIdx.x / kWarp] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
        uint32_t r = 0;
        for (int i = 0; i < kReadThreads / kWarp; ++i) r ^= s_fold[i];
        a.out[size_t(b) * size_t(a.split) + c] = bad ? ~0u : r;
    }
}

}  // namespace switchsd

extern "C" int switchsd_harness_read(const int32_t *ctx_tokens, const int32_t *ctx_lens, int32_t B, int32_t cap,
                                     const uint16_t *hidden, int32_t d, int32_t split, int32_t prefetch,
                                     uint32_t *out, void *stream) {
    if (!ctx_tokens || !ctx_lens || !hidden || !out) return SWITCHSD_ERR_ARG;
    if ((reinterpret_cast<uintptr_t>(ctx_tokens) & 15) != 0 || (reinterpret_cast<uintptr_t>(hidden) & 15) != 0 ||
        (reinterpret_cast<uintptr_t>(out) & 3) != 0)
        return SWITCHSD_ERR_ARG;
    if (B < 1 || B > 65535 || cap < 4 || cap % 4 != 0 || d < 8 || d % 8 != 0 || split < 1 || split > 1024)
        return SWITCHSD_ERR_SHAPE;
    static bool attr_done[64] = {false};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return SWITCHSD_ERR_CUDA;
    if (dev >= 0 && dev < 64 && !attr_done[dev]) {
        if (cudaFuncSetAttribute(read_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 int(kReadChunkWords * 16)) != cudaSuccess)
            return SWITCHSD_ERR_CUDA;
        attr_done[dev] = true;
    }
    // shared memory: the largest chunk any CTA can have
    const int64_t words = (int64_t(cap / 4) + split - 1) / split + (int64_t(d / 8) + split - 1) / split;
    const size_t smem = size_t(words < kReadChunkWords ? words : kReadChunkWords) * 16;
    ReadArgs a;
    a.ctx = ctx_tokens;
    a.lens = ctx_lens;
    a.hidden = hidden;
    a.out = out;
    a.B = B;
    a.cap = cap;
    a.d = d;
    a.split = split;
    a.prefetch = prefetch != 0;
    // an explicit cluster of one CTA, as for every kernel here that issues bulk copies
    const cudaError_t e = launch_pdl(read_kernel, dim3(unsigned(split), unsigned(B)), dim3(kReadThreads), smem,
                                     static_cast<cudaStream_t>(stream), 1u, a);
    return e == cudaSuccess ? SWITCHSD_OK : SWITCHSD_ERR_CUDA;
}
