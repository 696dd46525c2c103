/*
 * sc.h -- C ABI of the GB300 (sm_103a) verification step of speculative
 * cascades (Narasimhan et al., "Faster Cascades via Speculative Decoding").
 *
 * The library implements one call of GenSpecSample's verification phase
 * (Algorithm 4) with the SpecCascade target of Algorithm 5,
 *
 *     pi_j = (1 - delta_j) q_j + delta_j p_j                          (Eq. 6)
 *
 * where q_j = softmax(draft_logits[b, j] / T), p_j = softmax(target_logits[b, j] / T)
 * and delta_j is a deferral rule of Table 1 (with a token-specific rule of
 * Section 4.4, pi_j(v) = q_j(v) (1 - r_j(v)) + eta_j p_j(v) instead, see
 * SC_RULE_TOKEN_V1..3).  Per sequence b it accepts draft
 * token x_j when u[b, j] < min(1, pi_j(x_j) / q_j(x_j)), finds the first
 * rejection j*, and draws one new token from norm(max(0, pi_{j*} - q_{j*})),
 * or from pi_gamma := p_gamma (the drafter has no row at the bonus position)
 * when all gamma drafts are accepted.
 *
 * The same step with the vocabulary split across GPUs (a tensor-parallel LM
 * head) is declared in sc_shard.h.
 *
 * Conventions of every entry point:
 *  - All array pointers are CUDA device pointers owned by the caller.  The
 *    library allocates no device memory per call and never synchronises: work
 *    is queued on `stream` and results are valid once the stream reaches them.
 *  - Logits are row-major, contiguous, float32 or bf16 (raw 16-bit patterns).
 *  - CUDA graphs: a call may be captured into a graph (stream capture) once one
 *    call outside capture has run on the device with the same logit type and rule
 *    family (it configures the kernel); during capture the pointer arguments are
 *    only checked for NULL.  A replay reuses the captured workspace, which every
 *    call leaves ready for the next.
 *  - Synchronous argument errors return a negative sc_status and queue no work.
 *    Data errors found on the device never trap: they set bits in the optional
 *    `device_status` word (see SC_DEV_*) and the affected sequence receives the
 *    defined outputs num_accepted = 0, next_token = -1.
 *  - Limits: B, gamma, V >= 1; gamma <= SC_MAX_GAMMA; V <= sc_max_vocab(dtype);
 *    0 < T < inf, or T = 0 (greedy decoding) with a rule other than the token
 *    rules and lossy speculative decoding; 0 <= alpha <= 1 (the paper sweeps
 *    alpha over [0, 1]) for rules 0-8, 0 <= alpha < inf for rules 9-12 (a
 *    threshold on an entropy or a cross entropy, in nats).
 */
#ifndef SC_H_
#define SC_H_

#include <stddef.h>
#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum { SC_F32 = 0, SC_BF16 = 1 } sc_dtype;

/* Deferral rules delta(q, p) of Table 1 (strict inequalities as printed). */
typedef enum {
  SC_RULE_CHOW = 0,         /* max_v q(v) < 1 - alpha                           (Eq. 2)  */
  SC_RULE_DIFF = 1,         /* max_v q(v) < max_v p(v) - alpha                  (Eq. 5)  */
  SC_RULE_OPT = 2,          /* max_v q(v) < max_v p(v) - alpha * D_TV(p, q)     (Eq. 10) */
  SC_RULE_ALWAYS_DEFER = 3, /* delta = 1: standard speculative sampling, pi = p (Algorithm 1) */
  SC_RULE_NEVER_DEFER = 4,  /* delta = 0: pi = q, every draft is accepted */
  /* Token-specific targets (Section 4.4, TokenSpecCascade): a per-token deferral
   * r(v) in {0, 1}, eta = sum_v r(v) q(v) and pi(v) = q(v) (1 - r(v)) + eta p(v). */
  SC_RULE_TOKEN_V1 = 5,     /* r(v) = [q(v) < max p - alpha] */
  SC_RULE_TOKEN_V2 = 6,     /* r(v) = [p(v) < max p - alpha] */
  SC_RULE_TOKEN_V3 = 7,     /* r(v) = [p(v) < max p (1 - alpha)] */
  /* The other targets of Table 3, run through Algorithm 4 the same way. */
  SC_RULE_LOSSY = 8,        /* lossy speculative decoding: pi = max{min{q, p/(1 - alpha)}, p/beta}
                             * (pi need not sum to one; Lemma 2: the acceptance ratio is
                             * min(1, p(x)/((1 - alpha) q(x))), the residual norm(max(0, p/beta - q)));
                             * beta >= 1 - alpha, 1 for sc_verify and sc_verify_rows; with
                             * beta > 1 a rejection can leave the residual empty (p/beta <= q
                             * everywhere): no token is defined, next_token = -1 and
                             * num_accepted = j*, with no status bit */
  SC_RULE_BILD = 9,         /* BiLD*: delta = [D(q, p) > alpha], D(q, p) = -sum_v q(v) ln p(v) */
  /* Plug-in rules for the log loss (the paper's appendix on log loss), with
   * sum_v q ln q the negative entropy: */
  SC_RULE_CHOW_LOG = 10,    /* H(q) > alpha */
  SC_RULE_DIFF_LOG = 11,    /* sum q ln q < sum p ln p - alpha */
  SC_RULE_OPT_LOG = 12      /* sum q ln q < sum p ln p - alpha D_TV(p, q) */
} sc_rule;

typedef enum {
  SC_OK = 0,
  SC_ERR_INVALID_ARG = -1, /* a size, rule, alpha, T or pointer is out of its domain */
  SC_ERR_CUDA = -2,        /* the launch failed; cudaGetLastError() has the cause */
  SC_ERR_WORKSPACE = -3,   /* workspace missing or smaller than sc_workspace_bytes() */
  SC_ERR_UNSUPPORTED = -4, /* V too large for one thread-block cluster per row */
  SC_ERR_SCRATCH_LIMIT = -5 /* batch larger than sc_verify_static's built-in scratch */
} sc_status;

/* Bits of the optional device status word (OR-ed in, never cleared). */
#define SC_DEV_BAD_TOKEN 1u   /* a draft token outside [0, V) */
#define SC_DEV_BAD_LOGIT 2u   /* a NaN or +inf logit, or a row whose logits are all -inf */
#define SC_DEV_BAD_UNIFORM 4u /* a uniform outside [0, 1) */
#define SC_DEV_TIMEOUT 8u     /* an on-chip copy did not complete within the wait limit */

#define SC_MAX_GAMMA 255

/* Layout overrides, read from the environment at every call and meant for
 * measurements (the default layout is chosen from V, the batch and the SM count):
 *   SC_SLICE=n    logits per CTA slice of a row (n >= 64, rounded to a multiple of 8)
 *   SC_CLUSTER=c  CTAs per row pair (1 <= c <= 16; raised if the slices would not fit)
 *   SC_SPEC_RES=0|1  whether a rejected pair that is certainly row j* (every earlier
 *                 position of its slice reported without a rejection) stores its own
 *                 residual prefixes (default 1), or the owners always sample
 *   SC_POS_MAJOR=0|1 units in position-major order (default 1) or sequence-major
 *   SC_L2_HINT=n  copy all but the newest n chunks of a pair's slice, and every bonus
 *                 row, with the L2 evict-first policy (default 4; 0: no cache hints)
 *   SC_OPT_UB=0|1 whether OPT pairs accumulate the Bhattacharyya coefficient in
 *                 pass 1 for an upper bound on D_TV that settles band rows without
 *                 the TV pass (default: when C <= 4) */

/* Per-position diagnostics written by sc_verify_rows, [B][gamma+1][SC_ROW_FIELDS]
 * float32.  Position gamma (the bonus position) fills only MAXP and CAND. */
#define SC_ROW_MAXQ 0   /* max_v q_j(v) */
#define SC_ROW_MAXP 1   /* max_v p_j(v) */
#define SC_ROW_TV 2     /* D_TV(p_j, q_j) = sum_v max(0, p_j(v) - q_j(v)) (Lemma 3), or -1
                           when the decision did not need its exact value */
#define SC_ROW_DELTA 3  /* delta_j in {0, 1}; for a token rule r_j(x_j), the draft token's deferral */
#define SC_ROW_ACCEPT 4 /* a_j in {0, 1} (a_gamma = 0) */
#define SC_ROW_QX 5     /* q_j(x_j) */
#define SC_ROW_PIX 6    /* pi_j(x_j) */
#define SC_ROW_CAND 7   /* next_token at position j*, -1 at every other position */
#define SC_ROW_FIELDS 8

/* Device workspace needed by sc_verify for B sequences of gamma drafts
 * (independent of V).  Before its first use the workspace must be zeroed
 * (sc_workspace_init or a memset); every completed call leaves it zeroed again.
 * Calls that share one workspace must be ordered on one stream. */
size_t sc_workspace_bytes(int B, int gamma, int V);

/* Zero a workspace on `stream` (a cudaMemsetAsync). */
int sc_workspace_init(void *workspace, size_t workspace_bytes, cudaStream_t stream);

/* Largest supported vocabulary for a logit type. */
int sc_max_vocab(sc_dtype dtype);

/*
 * sc_verify -- one verification step (Algorithm 4 with Algorithm 5's target).
 *   draft_logits   [B][gamma][V]     q logits for the gamma drafted positions
 *   target_logits  [B][gamma+1][V]   p logits for positions 0..gamma
 *   draft_tokens   [B][gamma] int32  x_j, sampled by the drafter from q_j
 *   uniforms       [B][gamma+1] f32  u[b][j < gamma] is the Bernoulli draw of
 *                                    position j; u[b][gamma] is the single draw
 *                                    for the residual or bonus sample
 *   rule, alpha    deferral rule of Table 1 (or another rule of sc_rule) and its parameter
 *   temperature    T > 0: both q and p are softmax(logits / T).  T = 0 is greedy
 *                  decoding: the rule reads max q, max p and the entropies of
 *                  softmax(logits), and its D_TV is that of the one-hot q~, p~ at
 *                  the rows' argmaxes (lowest index on ties), 1(argmax q != argmax p);
 *                  pi = (1 - delta) q~ + delta p~, so a draft is rejected only when
 *                  delta = 1 and it is not the target's argmax, and the emitted
 *                  token at j* is the target's argmax (the uniforms are not read
 *                  for sampling)
 *   num_accepted   [B] int32 out: j* in [0, gamma]
 *   next_token     [B] int32 out: the token emitted at position j*.  The
 *                  emitted tokens of sequence b are draft_tokens[b][0 .. j*-1]
 *                  followed by next_token[b].
 *   workspace      sc_workspace_bytes(B, gamma, V) bytes, zeroed before first use
 *   device_status  optional int32 word receiving SC_DEV_* bits (may be NULL)
 * The residual and bonus draws are inverse-CDF samples in ascending vocabulary
 * order; the bonus position samples pi_gamma := p_gamma (no draft row exists there).
 */
int sc_verify(const void *draft_logits, const void *target_logits, sc_dtype dtype,
              const int32_t *draft_tokens, const float *uniforms, int B, int gamma, int V,
              sc_rule rule, float alpha, float temperature, int32_t *num_accepted,
              int32_t *next_token, void *workspace, size_t workspace_bytes,
              int32_t *device_status, cudaStream_t stream);

/* sc_verify that also writes the per-position diagnostics row_info
 * [B][gamma+1][SC_ROW_FIELDS] (row_info may be NULL, which equals sc_verify). */
int sc_verify_rows(const void *draft_logits, const void *target_logits, sc_dtype dtype,
                   const int32_t *draft_tokens, const float *uniforms, int B, int gamma, int V,
                   sc_rule rule, float alpha, float temperature, int32_t *num_accepted,
                   int32_t *next_token, void *workspace, size_t workspace_bytes,
                   int32_t *device_status, float *row_info, cudaStream_t stream);

/* sc_verify_rows with lossy speculative decoding's beta (Table 3): beta > 0 and
 * beta >= 1 - alpha when rule is SC_RULE_LOSSY, ignored otherwise. */
int sc_verify_ex(const void *draft_logits, const void *target_logits, sc_dtype dtype,
                 const int32_t *draft_tokens, const float *uniforms, int B, int gamma, int V,
                 sc_rule rule, float alpha, float beta, float temperature, int32_t *num_accepted,
                 int32_t *next_token, void *workspace, size_t workspace_bytes,
                 int32_t *device_status, float *row_info, cudaStream_t stream);

/*
 * sc_row_stats -- the per-position quantities the deferral rules of Table 1
 * read: max_v q_j(v), max_v p_j(v) and D_TV(p_j, q_j) (Lemma 3), for every pair
 * (b, j < gamma).  Outputs are [B*gamma] float32 each, index b*gamma + j.  A
 * row that is not a distribution (NaN / +inf logit, or all -inf) yields NaN.
 * target_logits has the same [B][gamma+1][V] layout as for sc_verify (the
 * bonus row is not read).
 */
int sc_row_stats(const void *draft_logits, const void *target_logits, sc_dtype dtype, int B,
                 int gamma, int V, float temperature, float *max_q, float *max_p, float *tv,
                 cudaStream_t stream);

/* Static description of an sc_status code. */
const char *sc_status_string(int code);

/* Builds with -DSC_DEBUG=1 check the kernel's computed indices, copy sizes and
 * alignments, skip an access that fails (its outputs are then undefined; a skipped
 * copy ends in SC_DEV_TIMEOUT) and record the kernel source line of the first
 * failure.  Returns that line (0: none), clearing it when `reset` is nonzero,
 * SC_ERR_CUDA if it cannot be read, and -1 in builds without the checks. */
int sc_debug_line(int reset);

/*
 * sc_verify_static -- sc_verify for callers that cannot allocate device memory.
 *
 * The paper has no counterpart: this entry point exists for code that must not
 * call cudaMalloc, e.g. an inference server whose device memory is carved up by
 * its own allocator before the first request, or a caller running where a
 * synchronising allocation would stall other streams.  Such callers still pass
 * their inputs and outputs, but need no workspace: the tickets, per-position
 * decision records and per-slice totals live in a fixed array compiled into the
 * library, one copy per device, held by every GPU that loads the library until
 * exit.
 *
 * Limits: B <= SC_STATIC_MAX_B and B * (gamma + 1) <= SC_STATIC_MAX_UNITS
 * (gamma >= 1, so at most SC_STATIC_MAX_UNITS / 2 = SC_STATIC_MAX_B sequences;
 * about 10.8 MiB of scratch); larger batches return SC_ERR_SCRATCH_LIMIT and
 * queue no work.  Other arguments are those of sc_verify and are checked the
 * same way, all before anything is queued.
 *
 * Every call looks up the array's device address in the current context; the
 * first call on a device also loads the library's module there, so make it
 * before any stream capture.  Every call clears the tickets it uses on `stream`
 * before launching.  All calls on a
 * device share the one array and it keeps the last call's contents, so calls that
 * may overlap on the GPU (different streams without ordering between them) race
 * and must not be issued; order them on one stream or serialise them.  Nothing is
 * allocated or freed by this call.
 */
#define SC_STATIC_MAX_B 2048
#define SC_STATIC_MAX_UNITS 4096
int sc_verify_static(const void *draft_logits, const void *target_logits, sc_dtype dtype,
                     const int32_t *draft_tokens, const float *uniforms, int B, int gamma, int V,
                     sc_rule rule, float alpha, float temperature, int32_t *num_accepted,
                     int32_t *next_token, int32_t *device_status, cudaStream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* SC_H_ */
