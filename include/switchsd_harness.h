/*
 * switchsd_harness.h -- device stand-in for the out-of-scope neural drafter and target model.
 *
 * Not part of the controller.  The paper's controller sits between a target-model forward and the
 * drafters (Fig. 1); both are outside this library.  Benchmarks and tests that drive the controller
 * step after step need the target's greedy tokens for each draft and a neural draft for the rows the
 * controller does not copy.  Greedy verification keeps each context equal to the target's own greedy
 * sequence, so the target is represented by that sequence: a caller-supplied token stream `future`
 * holding, for every row, the target's greedy tokens at absolute positions [L0, L0 + n_future).  The
 * same law is implemented on the host by the input generator package (synth.harness); both must
 * produce identical outputs.
 *
 * Randomness: word(seed, b, step, slot) = s(s(s(s(seed) ^ b) ^ step) ^ slot), where s is splitmix64
 * (Steele, Lea and Flood's finaliser with Vigna's published constants).  For draft index i the slots
 * are 4i + 0 (neural agreement coin, low 32 bits) and 4i + 1 (replacement token, (word >> 32) mod V).
 *
 * Per row b with L = ctx_lens[b] and g_i = future[b, L + i - L0] (0 outside [0, n_future)):
 *   - target[b, i] = g_i for i = 0..k;
 *   - mode[b] == SWITCHSD_MODE_COPY: vdraft = draft[b, 0..len), vlen = len = draft_len[b];
 *     otherwise a neural draft of gamma tokens: vdraft[i] = g_i if coin < thr_neural, else the
 *     replacement token, bumped by one (mod V) if it equals g_i; vlen = gamma;
 *   - vdraft is zero beyond vlen.
 *
 * Arrays (device, caller-owned): ctx_lens, mode, draft_len int32 [B]; draft int32 [B, k];
 * future int32 [B, n_future]; outputs vdraft int32 [B, k], vlen int32 [B], target int32 [B, k+1].
 * Returns SWITCHSD_OK, SWITCHSD_ERR_ARG, SWITCHSD_ERR_SHAPE or SWITCHSD_ERR_CUDA (codes of
 * switchsd.h).
 */
#ifndef SWITCHSD_HARNESS_H_
#define SWITCHSD_HARNESS_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct {
    int32_t B, k, V, L0, n_future, gamma, step;
    uint64_t seed;
    uint64_t thr_neural; /* threshold on a 32-bit word; 1 << 32 means always */
    void *stream;
    float p_hit, p_miss; /* sampled: target probability of a draft token equal to / different from the stream */
    float q_neural;      /* sampled: the neural drafter's probability of its token (copy drafts: 1) */
} switchsd_harness_params;

int switchsd_harness_target(const int32_t *ctx_lens, const int32_t *mode, const int32_t *draft,
                            const int32_t *draft_len, const int32_t *future, int32_t *vdraft,
                            int32_t *vlen, int32_t *target, const switchsd_harness_params *hp);

/*
 * The stand-in at temperature T > 0, feeding switchsd_verify_sampled.  vdraft / vlen as above; with
 * g[i] = future[L - L0 + i] and key(slot) = the harness key of (seed, row, step, slot):
 *   p[b][i]        p_hit if vdraft[i] == g[i] else p_miss (i < vlen; 0 beyond)
 *   q[b][i]        1 for a copy row, q_neural for a neural row (i < vlen; 1 beyond)
 *   u[b][i]        (key(4 i + 2) >> 40) * 2^-24, for every i < k (exact in binary32)
 *   resample[b][i] i < vlen: g[i], or when g[i] == vdraft[i] the token (key(4 i + 3) >> 32) mod V (plus
 *                  one mod V if that equals vdraft[i]) -- the residual excludes the rejected token;
 *                  i = vlen: g[vlen] (the bonus draw); 0 beyond.
 * p, q, u are float [B, k]; resample int32 [B, k+1].
 */
int switchsd_harness_sampled(const int32_t *ctx_lens, const int32_t *mode, const int32_t *draft,
                             const int32_t *draft_len, const int32_t *future, int32_t *vdraft, int32_t *vlen,
                             float *p, float *q, float *u, int32_t *resample, const switchsd_harness_params *hp);

/*
 * The stand-in for switchsd_verify_candidates.  A copy row's candidates (cand [B, W, D], cand_len
 * [B, W], ncand [B] from switchsd_step_candidates) are passed on; a neural row gets min(gamma, D)
 * neural tokens (the law of switchsd_harness_target) as its one candidate.  target[b][w][i] is the
 * stream's token at position L + i for every kept candidate (the target's greedy token after any prefix
 * the verification can accept), 0 for unused slots.  Outputs vcand [B, W, D], vlen [B, W], vn [B],
 * target [B, W, D+1].
 */
int switchsd_harness_candidates(const int32_t *ctx_lens, const int32_t *mode, const int32_t *cand,
                                const int32_t *cand_len, const int32_t *ncand, const int32_t *future, int32_t W,
                                int32_t D, int32_t *vcand, int32_t *vlen, int32_t *vn, int32_t *target,
                                const switchsd_harness_params *hp);

/*
 * Not a stand-in: the size-matched read ceiling that benchmarks set beside the step kernel.  Reads
 * what one step reads -- the first ctx_lens[b] tokens of every row (rounded up to whole 16-byte
 * words) and the hidden states -- and nothing else: grid (split, B) of 256-thread CTAs, CTA (c, b)
 * taking the c-th of `split` equal runs of row b's context words and of its d bf16 hidden values,
 * copied into shared memory by bulk (TMA) copies in chunks of up to 64 KB and xor-folded into
 * out[b * split + c] so no byte is left unread (~0u if a copy did not complete in time).  prefetch
 * != 0 issues the first chunk's copies before the kernel's grid-dependency wait (as the step kernel
 * does under SWITCHSD_PREFETCH_CONTEXT | SWITCHSD_PREFETCH_PROBE), else after it; launched with
 * programmatic stream serialization like every kernel of the library.
 * ctx_tokens int32 [B, cap] (16-byte aligned, cap a multiple of 4), ctx_lens int32 [B] (a length
 * outside [0, cap] reads nothing), hidden bf16 bits [B, d] (16-byte aligned, d a multiple of 8),
 * out uint32 [B * split]; split in [1, 1024].  Returns SWITCHSD_OK, SWITCHSD_ERR_ARG (NULL or
 * misaligned pointer), SWITCHSD_ERR_SHAPE or SWITCHSD_ERR_CUDA.
 */
int switchsd_harness_read(const int32_t *ctx_tokens, const int32_t *ctx_lens, int32_t B, int32_t cap,
                          const uint16_t *hidden, int32_t d, int32_t split, int32_t prefetch, uint32_t *out,
                          void *stream);

#ifdef __cplusplus
}
#endif

#endif /* SWITCHSD_HARNESS_H_ */
