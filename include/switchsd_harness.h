/*
 * switchsd_harness.h -- device stand-in for the out-of-scope neural drafter and target model.
 *
 * Not part of the controller.  The paper's controller sits between a target-model forward and the
 * drafters (Fig. 1); both are outside this library.  Benchmarks and tests that drive the controller
 * step after step need the target's greedy tokens for each draft, so this entry point synthesises
 * them on the device with a seeded per-token agreement law.  The same law is implemented on the host
 * by the input generator package (synth.harness) and both must produce identical outputs.
 *
 * Randomness: word(seed, b, step, slot) = s(s(s(s(seed) ^ b) ^ step) ^ slot), where s is splitmix64
 * (Steele, Lea and Flood's finaliser with Vigna's published constants).  For draft index i the slots
 * are 4i + 0 (agreement coin, low 32 bits), 4i + 1 (disagreeing token), 4i + 2 (neural draft token),
 * 4i + 3 (bonus token); a token is (word >> 32) mod V.
 *
 * Per row b with L = ctx_lens[b]:
 *   - mode[b] == SWITCHSD_MODE_COPY: the draft is draft[b, 0..len) with len = draft_len[b];
 *     otherwise a neural draft of k seeded tokens (len = k);
 *   - for i < len: agree iff i < agree_cap and coin < (labels[b, L + i - L0] ? thr_in : thr_out)
 *     (labels outside [0, n_labels) count as 0); target[i] = draft[i] if agree, else the seeded
 *     token, bumped by one (mod V) if it equals draft[i];
 *   - target[i] for i >= len is the seeded bonus token.
 *
 * Arrays (device, caller-owned): ctx_lens, mode, draft_len int32 [B]; draft int32 [B, k];
 * labels uint8 [B, n_labels]; outputs vdraft int32 [B, k] (zero beyond vlen), vlen int32 [B],
 * target int32 [B, k+1].  Returns SWITCHSD_OK, SWITCHSD_ERR_ARG, SWITCHSD_ERR_SHAPE or
 * SWITCHSD_ERR_CUDA (codes of switchsd.h).
 */
#ifndef SWITCHSD_HARNESS_H_
#define SWITCHSD_HARNESS_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct {
    int32_t B, k, V, L0, n_labels, agree_cap, step;
    uint64_t seed;
    uint64_t thr_in, thr_out; /* thresholds on a 32-bit word; 1 << 32 means always */
    void *stream;
} switchsd_harness_params;

int switchsd_harness_target(const int32_t *ctx_lens, const int32_t *mode, const int32_t *draft,
                            const int32_t *draft_len, const uint8_t *labels, int32_t *vdraft,
                            int32_t *vlen, int32_t *target, const switchsd_harness_params *hp);

#ifdef __cplusplus
}
#endif

#endif /* SWITCHSD_HARNESS_H_ */
