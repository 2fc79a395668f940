/*
 * switchsd.h -- C ABI of the SwitchSD per-step controller on one GB300 (sm_103a).
 *
 * SwitchSD ("To Copy or Not to Copy: Controlling Speculative Decoding via Intrinsic Model Signals")
 * decides after every verification step whether the next draft is copied from the context or left to
 * a neural drafter (Fig. 1).  This library runs that controller for B independent sequences:
 *
 *   switchsd_step    longest-suffix n-gram search (§3.3 kappa-gram gate, recency ranking), the
 *                    copy-intent probe logit (Eq. 3, or a two-layer extension), the three-way switch
 *                    (Fig. 1, Eq. 4) and the copy draft gather (§3.3 "Copy-Based Speculative
 *                    Generation");
 *   switchsd_verify  greedy verification and append (§3.3 "Parallel Verification", temperature 0 as
 *                    in App. A): accepted prefix length, then the accepted tokens and the target's own
 *                    next token are appended to the context;
 *   switchsd_verify_step  both, fused into one launch (verification of the previous draft, then the
 *                    next step).
 *
 * The target model and the neural drafter are outside the library; their outputs (hidden state at the
 * probed layer, the target's greedy tokens, the neural draft) arrive as arguments.
 *
 * General conventions
 *   - Every array pointer is a caller-owned DEVICE pointer (cudaMalloc / torch CUDA tensor memory) on
 *     the current CUDA device.  The library never frees or retains them.
 *   - Calls are asynchronous on `stream` (a cudaStream_t passed as void*; NULL = legacy default
 *     stream).  They return SWITCHSD_OK once the work is enqueued, or a negative host error code
 *     before anything is enqueued (bad argument, unsupported shape) or SWITCHSD_ERR_CUDA if a launch
 *     failed.  Outputs are valid once the stream reaches the call.
 *   - Per-row problems found on the device (bad length, capacity overflow) are reported in the
 *     optional per-row `status` array (SWITCHSD_ROW_*); the kernels never trap.
 *   - Token ids are opaque int32 values: only equality is used.
 *   - bf16 values are passed as their 16-bit patterns (uint16_t), the upper half of an IEEE binary32.
 *   - All calls may be captured into a CUDA graph: they allocate nothing and synchronise nothing
 *     (the host-staged entries switchsd_step_host / switchsd_verify_step_host synchronise when asked).
 */
#ifndef SWITCHSD_H_
#define SWITCHSD_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define SWITCHSD_ABI_VERSION 8

#define SWITCHSD_NMAX 32 /* largest supported n_max */
#define SWITCHSD_KMAX 64 /* largest supported draft length k */

/* Modes: the three cases of Fig. 1. */
#define SWITCHSD_MODE_NO_REP 0      /* (i) no repetition: neural draft */
#define SWITCHSD_MODE_COPY 1        /* (ii) repetition with copy intent: copy draft */
#define SWITCHSD_MODE_REP_NO_COPY 2 /* (iii) repetition without copy intent: neural draft */

/* Probe kinds. */
#define SWITCHSD_PROBE_LINEAR 0 /* Eq. 3: z = w^T h, probe_w = w[d] */
#define SWITCHSD_PROBE_MLP 1    /* z = w2 . ReLU(W1 h + b1) + b2, probe_w = W1[H1, d] then w2[H1] */

/* Host return codes. */
#define SWITCHSD_OK 0
#define SWITCHSD_ERR_ARG (-1)   /* NULL or misaligned pointer, bad enum */
#define SWITCHSD_ERR_SHAPE (-2) /* unsupported size */
#define SWITCHSD_ERR_CUDA (-3)  /* a CUDA call failed; cudaGetLastError() has the cause */

/* Per-row device status. */
#define SWITCHSD_ROW_OK 0
#define SWITCHSD_ROW_CAPACITY 1 /* verify: the append does not fit in cap; row left untouched */
#define SWITCHSD_ROW_BAD_LEN 2  /* ctx_lens[b] outside [1, cap] or draft_len[b] outside [0, k] */
#define SWITCHSD_ROW_TIMEOUT 3  /* an on-chip copy did not complete within its wait limit */

/* switchsd_params.prefetch bits. */
#define SWITCHSD_PREFETCH_CONTEXT 1
#define SWITCHSD_PREFETCH_PROBE 2

/* Slots of switchsd_params.counters. */
#define SWITCHSD_CTR_STEPS 0           /* + mode: rows whose step chose that mode (3 slots) */
#define SWITCHSD_CTR_COPY_DRAFTS 3     /* copy drafts verified */
#define SWITCHSD_CTR_COPY_ACCEPTED 4   /* their accepted tokens */
#define SWITCHSD_CTR_NEURAL_DRAFTS 5   /* other drafts verified */
#define SWITCHSD_CTR_NEURAL_ACCEPTED 6 /* their accepted tokens */
#define SWITCHSD_COUNTERS 7

/* Incremental n-gram index (switchsd_index_create); opaque. */
typedef struct switchsd_index switchsd_index;

/*
 * Parameters of switchsd_step.
 *
 *   B            number of rows (sequences), >= 1
 *   cap          row capacity in tokens (row stride of ctx_tokens), a multiple of 4, >= 4
 *   d            hidden size, a multiple of 8
 *   k            largest copy draft, 1..SWITCHSD_KMAX (the paper's D, App. D)
 *   n_min,n_max  n-gram lengths searched, 1 <= n_min <= n_max <= SWITCHSD_NMAX
 *   kappa        shortest match that may copy (§3.3, the paper sets 5); <= 0 means n_min
 *   logit_tau    decision threshold in logit space: copy iff z >= logit_tau (Eq. 4 with tau;
 *                tau = 0.5 gives 0.0; -INFINITY copies on every match, +INFINITY never copies)
 *   probe_kind   SWITCHSD_PROBE_LINEAR or SWITCHSD_PROBE_MLP
 *   probe_hidden H1 of the two-layer probe (1..1024); ignored for the linear probe.  The two-layer
 *                probe also needs d <= 8192 (its first layer runs on the tensor cores).
 *   b1, b2       two-layer probe biases: b1 device float[H1] or NULL (zero), b2 a float
 *   split        CTAs per row (1, 2, 4, 8 or 16); 0 lets the library choose
 *   workspace, workspace_bytes   device scratch for the two-layer probe: at least
 *                switchsd_workspace_bytes(params) bytes, 16-byte aligned, caller-owned; may be NULL for
 *                the linear probe.  It holds the first layer's split-K partial sums between the probe's
 *                kernel and the step kernel, so calls sharing one workspace must not overlap on the GPU
 *   index        NULL: search by rescanning the context.  Else an index from switchsd_index_create for
 *                the same B, cap, n_min and n_max, kept current by switchsd_index_build and by the
 *                verification entry points given the same index; the search then walks its chains
 *                (same results as the rescan).  Ignores split.
 *   out_match_n, out_match_end   optional device int32[B]: the winning match length n* and the end
 *                position e* of its most recent earlier occurrence (0 / -1 when none); may be NULL
 *   status       optional device int32[B] per-row status (SWITCHSD_ROW_*); may be NULL
 *   stream       cudaStream_t as void*
 *   prefetch     0, or a set of SWITCHSD_PREFETCH_* bits naming inputs that the rescan may start to read
 *                before the kernel that precedes the call on the stream has finished (programmatic
 *                dependent launch), so that their copies overlap that kernel's tail:
 *                  SWITCHSD_PREFETCH_CONTEXT  ctx_lens and ctx_tokens[b][0, ctx_lens[b])
 *                  SWITCHSD_PREFETCH_PROBE    hidden and the linear probe's weights
 *                For every bit set the caller promises that (a) the kernel immediately before this
 *                call on the stream does not write those inputs, and (b) if that kernel was itself
 *                launched with programmatic stream serialization, it waits for its own predecessors
 *                (griddepcontrol.wait) before it lets dependents start -- every kernel of this library
 *                does, and a kernel launched without that attribute always does.  The earlier writer
 *                of those inputs is then complete when the copies start.  A copy or memset just before
 *                the call is always safe.  In a serving loop the target's last kernel (its argmax)
 *                writes neither the context nor the hidden state.  The previous draft, its length
 *                and the target argmax are always read after the wait.  The index search reads the
 *                row's length and tail (CONTEXT) and computes the linear probe (PROBE) before the wait;
 *                its tables come after it.  With the two-layer probe SWITCHSD_PREFETCH_PROBE lets the
 *                probe kernel's copies of the hidden states and W1 and its MMAs start early, and that
 *                kernel then releases the call's step kernel at once (whose reads before its own wait
 *                are still only those the bits name; its wait covers the probe kernel, whose stores
 *                follow that kernel's wait).  A call's kernels write the workspace, the outputs and, when
 *                verifying, the context and lengths; the call's last kernel may release the next kernel
 *                on the stream before the first-layer probe kernel of the same call has finished, which
 *                writes only the workspace.  Other bits are SWITCHSD_ERR_ARG.
 *   hidden_rows  0 or 1: hidden is [B, d], the state the probe reads for each row.  k + 1 (the fused
 *                switchsd_verify_step and switchsd_verify_sampled_step only): hidden is the
 *                target's verification output [B, k+1, d] and the probe reads row a_b of each row b --
 *                the state that produced the appended token t[a_b], the most recent one the target
 *                computed -- or row 0 when nothing was appended (capacity, bad lengths).  The probe's
 *                copies then wait for the verification; SWITCHSD_PREFETCH_PROBE is ignored.  With the
 *                two-layer probe a gather kernel first copies each row's a_b state (by the same
 *                acceptance rule) into the workspace, which switchsd_workspace_bytes then sizes for it.
 *                Any other value is SWITCHSD_ERR_ARG.
 *   len_bound    0, or an upper bound on every ctx_lens[b] before the call's append (<= cap).  The rescan
 *                then splits each row's ends between its CTAs on the bound instead of on the row's
 *                length, so the context copies leave before the length is read; a row longer than the
 *                bound gets SWITCHSD_ROW_BAD_LEN.  cap is always a valid bound; a bound far above the
 *                lengths leaves CTAs idle and copies bytes past the rows' ends.  The index search
 *                ignores it.  Outside [0, cap]: SWITCHSD_ERR_ARG.
 *   counters     optional device uint64[SWITCHSD_COUNTERS], or NULL: the controller's per-mode tallies
 *                (the paper's copy-iteration share and mean accepted length per drafter, §4 and Table
 *                1), added to by every row of every call -- the caller zeroes them when it wants to
 *                start counting:
 *                  [SWITCHSD_CTR_STEPS + m]  rows whose step chose mode m (SWITCHSD_MODE_*)
 *                  [SWITCHSD_CTR_COPY_DRAFTS], [SWITCHSD_CTR_COPY_ACCEPTED]  drafts verified whose
 *                        previous step was COPY, and the tokens accepted of them
 *                  [SWITCHSD_CTR_NEURAL_DRAFTS], [SWITCHSD_CTR_NEURAL_ACCEPTED]  the same for the
 *                        other drafts (the neural drafter's)
 *                The fused verifications take each row's previous mode from out_mode[b] as the call
 *                finds it (the caller passes the same out_mode array every step; the call overwrites it
 *                with the new mode).  Rows whose verification fails (bad length, capacity) add no draft.
 *                Integer additions: the totals do not depend on the order of the rows.  The candidate
 *                entry points ignore it.
 */
typedef struct {
    int32_t B, cap, d, k, n_min, n_max, kappa;
    float logit_tau;
    int32_t probe_kind;
    int32_t probe_hidden;
    const float *b1;
    float b2;
    int32_t split;
    void *workspace;
    size_t workspace_bytes;
    switchsd_index *index;
    int32_t *out_match_n;
    int32_t *out_match_end;
    int32_t *status;
    void *stream;
    int32_t prefetch;
    int32_t hidden_rows;
    int32_t len_bound;
    uint64_t *counters;
} switchsd_params;

/*
 * One controller step for B rows (§3.3, Fig. 1).
 *
 *   ctx_tokens  int32 [B, cap] row-major, 16-byte aligned; row b holds its context x[0..L_b-1]
 *   ctx_lens    int32 [B]; L_b = ctx_lens[b], 1 <= L_b <= cap
 *   hidden      bf16 [B, d] row-major, 16-byte aligned: the target model's hidden state at the probed
 *               layer for the row's current (last) token
 *   probe_w     bf16, 16-byte aligned: w[d] (linear) or W1[H1, d] row-major followed by w2[H1]
 *
 * For each row: (n*, e*) = the longest n in [n_min, n_max] whose suffix x[L-n..L-1] also ends at an
 * earlier position e <= L-2, and for that n the most recent such e.  z = the probe logit (fp32
 * accumulation of bf16 products).  mode = NO_REP if no match, COPY if n* >= kappa and
 * z >= logit_tau, else REP_NO_COPY.  For COPY rows the draft is x[e*+1 .. e*+len] with
 * len = min(k, L-1-e*); other rows get len 0 (the caller's neural drafter takes over).
 *
 *   out_draft   int32 [B, k]: entries at and beyond out_len[b] are unspecified
 *   out_len     int32 [B]
 *   out_mode    int32 [B]   (SWITCHSD_MODE_*)
 *   out_score   float [B]   the probe logit z (written for every row)
 *
 * Rows with a bad length get mode NO_REP, len 0 and status SWITCHSD_ROW_BAD_LEN.
 */
int switchsd_step(const int32_t *ctx_tokens, const int32_t *ctx_lens, const uint16_t *hidden,
                  const uint16_t *probe_w, const switchsd_params *params, int32_t *out_draft,
                  int32_t *out_len, int32_t *out_mode, float *out_score);

/*
 * Parameters of switchsd_verify.
 *
 *   B, cap, k    as for switchsd_step
 *   draft_len    device int32 [B]: tokens of the draft to verify per row, 0..k (a copy row passes
 *                switchsd_step's out_len, a neural row its own draft length)
 *   ctx_tokens   device int32 [B, cap] (modified: accepted tokens are appended)
 *   ctx_lens     device int32 [B]      (modified: grows by accepted + 1)
 *   status       optional device int32 [B]; may be NULL
 *   index        NULL, or the row index (see switchsd_params): the appended positions are inserted
 *   stream       cudaStream_t as void*
 */
typedef struct {
    int32_t B, cap, k;
    const int32_t *draft_len;
    int32_t *ctx_tokens;
    int32_t *ctx_lens;
    int32_t *status;
    switchsd_index *index;
    void *stream;
} switchsd_verify_params;

/*
 * Greedy verification and append (§3.3 "Parallel Verification", temperature 0, App. A).
 *
 *   draft          int32 [B, k]: the draft that was verified (copy or neural)
 *   target_argmax  int32 [B, k+1]: the target model's greedy token after each draft prefix; entry i
 *                  is its prediction for the position of draft[i], entry len its next token after a
 *                  fully accepted draft
 *   out_accept     int32 [B]: a = number of leading draft tokens equal to target_argmax
 *
 * The row's context receives draft[0..a) then target_argmax[a]; ctx_lens grows by a+1.  If that does
 * not fit in cap, the row is untouched, out_accept = -1 and status = SWITCHSD_ROW_CAPACITY.
 */
int switchsd_verify(const int32_t *draft, const int32_t *target_argmax, int32_t *out_accept,
                    const switchsd_verify_params *vp);

/*
 * Verification and append at temperature T > 0 (App. A runs SwitchSD with sampling; the acceptance
 * rule is the speculative-sampling rule of the works §2 builds on).  Draft token i is accepted iff
 * u[i] * q[i] < p[i], the product rounded to binary32 and compared in binary32: the event
 * u < min(1, p / q) for u uniform in [0, 1).  A copy draft is deterministic (q = 1), so a copied token
 * is accepted with the target's probability of it.
 *
 *   draft      int32 [B, k]: the draft that was verified (copy or neural)
 *   p_draft    float [B, k]: the target's probability of draft[i] at its position
 *   q_draft    float [B, k]: the drafter's probability of draft[i], or NULL when every row holds a copy
 *              draft (q = 1); a copy row among neural rows passes 1.0 entries
 *   u          float [B, k]: uniform draws in [0, 1), one per draft position (the caller's random numbers)
 *   resample   int32 [B, k+1]: entry a is the token appended after a acceptances: for a < len the
 *              caller's draw from the residual distribution max(0, p - q) renormalised at that position,
 *              for a = len its draw from the target after the full draft
 *   out_accept int32 [B]: a, the accepted length
 *
 * The row's context receives draft[0..a) then resample[a]; ctx_lens grows by a+1; capacity, status and
 * bad lengths as switchsd_verify.  With p one-hot (T -> 0) and resample = the argmax this is
 * switchsd_verify.  With vp->index the index kernel applies the same rule and inserts the appended
 * positions, as for switchsd_verify.
 */
int switchsd_verify_sampled(const int32_t *draft, const float *p_draft, const float *q_draft, const float *u,
                            const int32_t *resample, int32_t *out_accept, const switchsd_verify_params *vp);

/*
 * One controller iteration in one launch (§3.3 "Overall Framework": after every verification step the
 * controller decides the next draft, Fig. 1): greedy verification and append of the previous draft,
 * exactly as switchsd_verify, then switchsd_step on the extended context.  The result equals
 * switchsd_verify followed by switchsd_step with the same arguments, at the cost of one launch.
 *
 *   draft, target_argmax, draft_len  the previous iteration's verified draft, as for switchsd_verify
 *                 (device int32 [B, k], [B, k+1], [B])
 *   out_accept    device int32 [B]: accepted length a, or -1 if the append did not fit / bad lengths
 *   ctx_tokens, ctx_lens   device, modified in place by the append, then searched by the step
 *   hidden, probe_w, params, out_draft, out_len, out_mode, out_score   as for switchsd_step
 *
 * params->status receives SWITCHSD_ROW_CAPACITY when the append did not fit (the step then runs on
 * the unchanged context), SWITCHSD_ROW_BAD_LEN for a bad ctx_lens[b] or draft_len[b], else the step's
 * status.  The draft buffers must not alias out_draft.
 */
int switchsd_verify_step(const int32_t *draft, const int32_t *target_argmax, const int32_t *draft_len,
                         int32_t *out_accept, int32_t *ctx_tokens, int32_t *ctx_lens,
                         const uint16_t *hidden, const uint16_t *probe_w,
                         const switchsd_params *params, int32_t *out_draft, int32_t *out_len,
                         int32_t *out_mode, float *out_score);

/*
 * switchsd_verify_step at temperature T > 0: the sampled verification and append of the previous draft,
 * exactly as switchsd_verify_sampled (same arguments: draft, p_draft, q_draft or NULL, u, resample,
 * draft_len), then switchsd_step on the extended context, in one launch (with params->index, in the
 * index kernel).  Statuses as switchsd_verify_step.
 */
int switchsd_verify_sampled_step(const int32_t *draft, const float *p_draft, const float *q_draft, const float *u,
                                 const int32_t *resample, const int32_t *draft_len, int32_t *out_accept,
                                 int32_t *ctx_tokens, int32_t *ctx_lens, const uint16_t *hidden,
                                 const uint16_t *probe_w, const switchsd_params *params, int32_t *out_draft,
                                 int32_t *out_len, int32_t *out_mode, float *out_score);

/*
 * Host staging around one step: switchsd_step / switchsd_verify_step for inputs that arrive in host
 * memory and results read back on the host, in one call.  Before the step, in_bytes are copied from
 * in_host to in_dev (device; typically the hidden states the step then reads); after it, out_bytes
 * from out_dev (device; typically one buffer holding the step's mode, draft length, accepted length
 * and draft) to out_host.  Both copies run on params->stream, ordered with the step: for page-locked
 * host memory mapped into the device's address space (any pinned allocation under unified addressing)
 * as a small kernel that reads or writes the host buffer through its device address, otherwise as
 * cudaMemcpyAsync.  After an input copy by kernel the step keeps a SWITCHSD_PREFETCH_* bit only if
 * the copied range misses the inputs that bit covers.  A zero byte count skips that copy.  synchronize != 0: the call returns after the stream has drained, so out_host holds the
 * results; 0: everything is queued on the stream and the call returns at once.
 */
typedef struct {
    const void *in_host;
    void *in_dev;
    size_t in_bytes;
    const void *out_dev;
    void *out_host;
    size_t out_bytes;
    int32_t synchronize;
} switchsd_host_io;

/* switchsd_step between the two copies of `io`.  Returns SWITCHSD_ERR_ARG for a NULL io or params or a
 * NULL pointer of a copy with a nonzero byte count, SWITCHSD_ERR_CUDA when a copy or the
 * synchronisation fails, else switchsd_step's code (a step that fails validation queues no copy back). */
int switchsd_step_host(const switchsd_host_io *io, const int32_t *ctx_tokens, const int32_t *ctx_lens,
                       const uint16_t *hidden, const uint16_t *probe_w, const switchsd_params *params,
                       int32_t *out_draft, int32_t *out_len, int32_t *out_mode, float *out_score);

/* switchsd_verify_step between the two copies of `io`; codes as switchsd_step_host. */
int switchsd_verify_step_host(const switchsd_host_io *io, const int32_t *draft, const int32_t *target_argmax,
                              const int32_t *draft_len, int32_t *out_accept, int32_t *ctx_tokens,
                              int32_t *ctx_lens, const uint16_t *hidden, const uint16_t *probe_w,
                              const switchsd_params *params, int32_t *out_draft, int32_t *out_len,
                              int32_t *out_mode, float *out_score);

/* switchsd_verify_sampled_step between the two copies of `io`; codes as switchsd_step_host. */
int switchsd_verify_sampled_step_host(const switchsd_host_io *io, const int32_t *draft, const float *p_draft,
                                      const float *q_draft, const float *u, const int32_t *resample,
                                      const int32_t *draft_len, int32_t *out_accept, int32_t *ctx_tokens,
                                      int32_t *ctx_lens, const uint16_t *hidden, const uint16_t *probe_w,
                                      const switchsd_params *params, int32_t *out_draft, int32_t *out_len,
                                      int32_t *out_mode, float *out_score);

/*
 * The arguments of one switchsd_verify_step call (draft, target_argmax and draft_len all set), of one
 * switchsd_verify_sampled_step call (p_draft and u set as well -- q_draft may stay NULL -- and
 * target_argmax holding the resample tokens), or of one switchsd_step call (the verification buffers
 * all NULL; out_accept is then unused), for switchsd_plan_create.
 */
typedef struct {
    const int32_t *draft, *target_argmax, *draft_len;
    int32_t *out_accept;
    int32_t *ctx_tokens, *ctx_lens;
    const uint16_t *hidden, *probe_w;
    const switchsd_params *params;
    int32_t *out_draft, *out_len, *out_mode;
    float *out_score;
    const float *p_draft, *q_draft, *u;
} switchsd_step_args;

/* A host-staged step recorded once as a CUDA graph (opaque). */
typedef struct switchsd_plan switchsd_plan;

/*
 * Records what switchsd_verify_step_host (or switchsd_step_host) does with `args` and `io` -- the H2D
 * copy, the step's launch(es), the D2H copy -- into a CUDA graph, by stream capture on a private
 * stream; nothing runs.  io->synchronize is ignored (switchsd_plan_run takes it).  The recorded
 * launches hold the device pointers and the parameter values, so *args and *args->params may be freed
 * after the call; replays launch on args->params->stream.  The caller keeps every buffer alive and, for
 * the two-layer probe, the workspace unshared while the plan can run.  Returns SWITCHSD_ERR_ARG (NULL
 * out, args, params or io, a partial set of verification buffers, p_draft without u, a copy without
 * buffers), SWITCHSD_ERR_CUDA (capture or instantiation failed), or the step's own validation code;
 * *out is then NULL.
 */
int switchsd_plan_create(const switchsd_step_args *args, const switchsd_host_io *io, switchsd_plan **out);

/*
 * Replays the plan on its stream.  in_host / out_host: the host ends of the two copies for this
 * replay (NULL: the ones of the last replay, first those of io at creation); the device ends and byte
 * counts are fixed, and a copy recorded as a kernel (pinned buffer at creation) takes pinned buffers
 * only.  synchronize != 0: returns after the stream has drained.  Equivalent to the switchsd_*_host
 * call it recorded.  SWITCHSD_ERR_ARG for a NULL plan or a pageable buffer where a pinned one was
 * recorded, SWITCHSD_ERR_CUDA if a copy could not be retargeted or the launch or synchronisation
 * failed.
 */
int switchsd_plan_run(switchsd_plan *plan, const void *in_host, void *out_host, int32_t synchronize);

/* Frees the plan's graph (NULL is ignored).  The plan must not be running. */
void switchsd_plan_destroy(switchsd_plan *plan);

/*
 * Bytes of device workspace switchsd_step / switchsd_verify_step need for `params` (0 for the linear
 * probe; for the two-layer probe, S x B x H1p floats rounded up to 256 bytes, where S is the first
 * layer's split of d -- the largest power of two <= 16 with at least two 64-element chunks of d per
 * part, 16 for d >= 2048 -- and H1p is probe_hidden rounded up to 64; with hidden_rows > 1, B x d bf16
 * more, rounded up to 256 bytes, for the gathered states).  Reads B, d, probe_kind, probe_hidden and
 * hidden_rows only.
 */
size_t switchsd_workspace_bytes(const switchsd_params *params);

/*
 * switchsd_step for callers that cannot allocate device memory.  The paper has no counterpart: this is
 * a convenience of the library.  Some callers cannot hand the library a workspace at call time (an
 * inference server that gives all of the GPU's memory to its own pool when it starts, or a host program
 * with no CUDA allocator of its own); this entry point takes the same arguments as switchsd_step, ignores
 * params->workspace and uses a fixed 16 MiB array compiled into the library instead.  It allocates
 * nothing (no cudaMalloc, no cudaFree).
 *
 *   Limit: the two-layer probe needs switchsd_workspace_bytes(params) <= 16 MiB (S x B x H1p <= 4 Mi
 *   floats: for example B <= 1,024 with d >= 2048 and 256 hidden units); larger requests return
 *   SWITCHSD_ERR_SHAPE.  The linear probe has no limit beyond switchsd_step's.  Like switchsd_step it
 *   verifies nothing, so params->hidden_rows must be 0 or 1.
 *   Set-up: the first call on each device looks up the array's device address (cudaGetSymbolAddress,
 *   with that device current) and keeps it; make that first call before any stream capture.  A device
 *   reset (cudaDeviceReset) invalidates the kept address: do not call this entry point on a device after
 *   resetting it in the same process.
 *   Sharing: every call on a device uses the same array, and the array keeps whatever the last call
 *   left there.  Nothing in it needs to start at zero (each call writes every entry it reads), but calls
 *   that overlap on the GPU race on it: issue them on one stream, or order them.
 *   Every GPU that loads the library holds the array until the process exits.
 */
int switchsd_step_static_workspace(const int32_t *ctx_tokens, const int32_t *ctx_lens,
                                   const uint16_t *hidden, const uint16_t *probe_w,
                                   const switchsd_params *params, int32_t *out_draft,
                                   int32_t *out_len, int32_t *out_mode, float *out_score);

/*
 * Incremental n-gram index: the search of §3.3 without rescanning the context.  Not in the paper (it
 * states only the search's result); the index returns exactly the rescan's (n*, e*).
 *
 * For every row and every n in [n_min, n_max] it keeps hash heads (the most recent end position of
 * each bucket of n-grams, at least 2 cap buckets) and a chain of previous end positions per bucket.
 * A lookup walks the suffix's chain from the most recent entry and verifies candidates token by token,
 * so collisions cost time, never correctness.  Appended tokens are inserted by switchsd_verify and
 * switchsd_verify_step when their params carry the index.
 *
 *   switchsd_index_create   allocates the index for params' B, cap, n_min, n_max (device memory, the
 *                           library's only allocation: see switchsd_index_bytes); SWITCHSD_ERR_CUDA if
 *                           the allocation fails.  The index belongs to the current device.
 *   switchsd_index_build    (re)builds it from ctx_tokens / ctx_lens on `stream` (asynchronous); call
 *                           it once for the initial contexts and after any change made outside the
 *                           library's verification entry points.  Lowering ctx_lens and appending the
 *                           same tokens again needs no rebuild (those insertions are no-ops); appending
 *                           different tokens after lowering ctx_lens does.
 *   switchsd_index_bytes    device bytes the index holds.
 *   switchsd_index_destroy  frees it (NULL is a no-op); no call using it may still be in flight.
 */
int switchsd_index_create(const switchsd_params *params, switchsd_index **out);
int switchsd_index_build(switchsd_index *index, const int32_t *ctx_tokens, const int32_t *ctx_lens,
                         void *stream);
size_t switchsd_index_bytes(const switchsd_index *index);
void switchsd_index_destroy(switchsd_index *index);

/* Human-readable text of a host return code or a row status (static storage, never NULL). */
const char *switchsd_strerror(int code);

#define SWITCHSD_WMAX 16 /* largest number of copy candidates W */

/*
 * The step with W copy candidates (§3.3 "Copy-Based Speculative Generation": up to W continuations of
 * length D retrieved from the context, ranked by recency; App. D uses W = 10, D = 20).  The candidates
 * are the W most recent ends e <= L-2 at which the kappa-gram ending at the current token recurs (the
 * common suffix is at least kappa = params->kappa, or n_min when <= 0, tokens long), most recent first;
 * candidate w continues with x[e_w+1 .. e_w+len_w], len_w = min(D, L-1-e_w).  The mode: no repetition
 * when no n_min-gram of the suffix recurs, copy when a candidate exists and z >= logit_tau, repetition
 * without copy otherwise.  Everything else as switchsd_step (params->k is only the bound of the staged
 * look-ahead and must be >= 1).  With params->index the index kernel lists the ends from its chain of
 * the kappa-gram, so kappa (or n_min when <= 0) must be at least the index's n_min
 * (SWITCHSD_ERR_SHAPE otherwise); a kappa above n_max gives no candidate, as for the rescan.
 *
 *   W, D          1..SWITCHSD_WMAX, 1..SWITCHSD_KMAX
 *   out_cand      device int32 [B, W, D]: candidate w's tokens in [b][w][0, len_w)
 *   out_cand_len  device int32 [B, W]: len_w for w < ncand
 *   out_ncand     device int32 [B]: candidates of a copy row (0 for the other modes)
 *   out_mode, out_score   as switchsd_step (out_match_n / out_match_end / status from params as well)
 */
int switchsd_step_candidates(const int32_t *ctx_tokens, const int32_t *ctx_lens, const uint16_t *hidden,
                             const uint16_t *probe_w, const switchsd_params *params, int32_t W, int32_t D,
                             int32_t *out_cand, int32_t *out_cand_len, int32_t *out_ncand, int32_t *out_mode,
                             float *out_score);

/*
 * Parameters of switchsd_verify_candidates.
 *
 *   B, cap        as switchsd_verify_params;  W, D  the candidate slots (as switchsd_step_candidates)
 *   cand_len      device int32 [B, W], ncand device int32 [B] (a neural row passes its draft as the one
 *                 candidate; ncand = 0 counts as one empty candidate)
 *   ctx_tokens, ctx_lens, status, stream, index   as switchsd_verify_params (with an index the index
 *                 kernel verifies, appends and inserts the appended positions)
 */
typedef struct {
    int32_t B, cap, W, D;
    const int32_t *cand_len;
    const int32_t *ncand;
    int32_t *ctx_tokens;
    int32_t *ctx_lens;
    int32_t *status;
    void *stream;
    switchsd_index *index;  /* NULL, or the index kept current by the append (as switchsd_verify_params) */
} switchsd_candidates_verify_params;

/*
 * Verification of the W candidates of each row (§3.3 "Parallel Verification with Block-Triangular
 * Attention": one target pass checks every candidate, and the longest validated continuation is kept).
 *
 *   cand        device int32 [B, W, D]
 *   target      device int32 [B, W, D+1]: the target's greedy token after each prefix of candidate w
 *   out_accept  device int32 [B]: the kept candidate's accepted length a (-1: capacity / bad lengths)
 *   out_choice  device int32 [B]: the kept candidate (the longest accepted, the lowest index on a tie)
 *
 * The row receives the kept candidate's a tokens, then its target token at a; ctx_lens grows by a+1.
 * Capacity and bad lengths as switchsd_verify.
 */
int switchsd_verify_candidates(const int32_t *cand, const int32_t *target, int32_t *out_accept, int32_t *out_choice,
                               const switchsd_candidates_verify_params *vp);

/*
 * switchsd_verify_candidates then switchsd_step_candidates in one launch (§3.3 "Overall Framework"):
 * the previous iteration's W candidates (cand [B, W, D], target [B, W, D+1], cand_len [B, W], ncand
 * [B], as switchsd_verify_candidates) are verified and the kept one appended, then the next
 * candidates are searched on the extended context.  out_accept / out_choice as
 * switchsd_verify_candidates; the other arguments as switchsd_step_candidates (the verified and the new
 * candidate buffers must not alias).  params->status: as switchsd_verify_step.
 */
int switchsd_verify_candidates_step(const int32_t *cand, const int32_t *target, const int32_t *cand_len,
                                    const int32_t *ncand, int32_t *out_accept, int32_t *out_choice,
                                    int32_t *ctx_tokens, int32_t *ctx_lens, const uint16_t *hidden,
                                    const uint16_t *probe_w, const switchsd_params *params, int32_t W, int32_t D,
                                    int32_t *out_cand, int32_t *out_cand_len, int32_t *out_ncand, int32_t *out_mode,
                                    float *out_score);

/*
 * Copy-mode labels (§3.2, "Problem Formulation"): the probe's training labels.  Position j of row b is
 * labelled 1 when it lies in a window of n consecutive tokens that also occurs starting at an earlier
 * position of the row (the paper uses n = n_train = 5); every other position 0.  The same exact token
 * comparisons as the search, over every position instead of the current one.
 *
 *   ctx_tokens  device int32 [B, cap], ctx_lens device int32 [B] (a length outside [0, cap] labels
 *               nothing)
 *   n           1..SWITCHSD_NMAX
 *   out_labels  device uint8 [B, cap]: 0 / 1 for j < ctx_lens[b], 0 beyond
 *   workspace   device scratch of at least switchsd_labels_workspace_bytes(B, cap) bytes, 4-byte
 *               aligned, caller-owned (a first-occurrence table per row and the table slot of every
 *               window start; calls sharing it must not overlap on the GPU)
 *   stream      cudaStream_t as void*
 */
size_t switchsd_labels_workspace_bytes(int32_t B, int32_t cap);
int switchsd_copy_labels(const int32_t *ctx_tokens, const int32_t *ctx_lens, int32_t B, int32_t cap, int32_t n,
                         uint8_t *out_labels, void *workspace, size_t workspace_bytes, void *stream);

/* SWITCHSD_ABI_VERSION of the loaded library. */
int switchsd_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* SWITCHSD_H_ */
