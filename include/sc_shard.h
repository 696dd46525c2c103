/*
 * sc_shard.h -- the verification step of speculative cascades with the
 * vocabulary split across W GPUs (a tensor-parallel LM head: GPU r holds the
 * logits of the tokens [shard_begin[r], shard_begin[r+1]) of every row).
 *
 * It computes exactly what sc_verify computes (Algorithm 4 with Algorithm 5's
 * target pi = (1 - delta) q + delta p, Eq. 6, for the deferral rules of Table 1
 * and SpecDecode's delta = 1), with the reductions over the vocabulary that
 * sc_verify does inside one thread-block cluster done in two levels: inside
 * each GPU, then across GPUs through small messages that the caller exchanges
 * with an all-gather (e.g. NCCL): four, five with SC_RULE_OPT.  No logit ever
 * leaves its GPU.
 *
 * One step on every rank r, in this order (the caller all-gathers each
 * message in rank order between the calls):
 *
 *   sc_shard_pass1   pass 1 over the local logits: per row the rank's
 *                    (max logit, sum of exponentials), the logits of each
 *                    draft token the rank holds, and with SC_RULE_OPT the
 *                    pair's Bhattacharyya sum (Hellinger's upper bound on
 *                    D_TV)                                     -> message 1
 *   sc_shard_decide  merges the W messages 1 (the same arithmetic in the same
 *                    order on every rank, so every rank takes the same
 *                    decisions): M, S, max q and max p of every row, delta
 *                    (Table 1) and the acceptance test (Algorithm 4).  With
 *                    SC_RULE_OPT a pair inside the band
 *                    max p - alpha <= max q < max p needs D_TV (Eq. 10):
 *                    where the upper bound does not settle delta, the rank
 *                    sends its part of a lower bound on D_TV  -> message 2 (OPT)
 *   sc_shard_tv      (SC_RULE_OPT only) sums the W parts of the lower bound;
 *                    where it does not settle delta = 0 either, the rank sums
 *                    its part of the residual weights (Lemma 3) -> message 3 (OPT)
 *   sc_shard_accept  merges the W messages 3, finishes delta and acceptance
 *                    of the band pairs, settles j* = min{j : a_j = 0}, and
 *                    sums the rank's part of the weights of the row it draws
 *                    from: norm(max(0, p - q)) of row j*, or p of the bonus
 *                    row when j* = gamma                      -> message 4
 *   sc_shard_draw    finds the rank, slice and segment holding u R (the
 *                    inverse CDF in ascending token order, u = uniforms[b][gamma]);
 *                    that rank draws the token, the others send -1
 *                                                              -> message 5
 *   sc_shard_finish  merges the W messages 5 into num_accepted and next_token
 *                    (identical on every rank).
 *
 * Conventions are those of sc.h: device pointers owned by the caller, work
 * queued on `stream`, nothing allocated and nothing synchronised; argument
 * errors return a negative sc_status before anything is queued; data errors
 * set SC_DEV_* bits in the optional device_status word and give the sequence
 * num_accepted = 0, next_token = -1.
 *
 * Shared arguments:
 *   draft_shard    [B][gamma][ld] logits (float32 or bf16): element v - shard_begin[rank]
 *                  of row (b, j) is the logit of token v; only the first
 *                  shard_begin[rank+1] - shard_begin[rank] of each row are read
 *   target_shard   [B][gamma+1][ld], the same layout
 *   ld             elements between consecutive rows (>= the shard's width).  Rows
 *                  whose start is 16-byte aligned (base and ld * element size) are
 *                  read with vector loads, others element by element
 *   W, rank        1 <= W <= SC_SHARD_MAX, 0 <= rank < W
 *   shard_begin    HOST array of W + 1 token indices, 0 = shard_begin[0] <
 *                  shard_begin[1] < ... < shard_begin[W] = V (every shard nonempty)
 *   workspace      sc_shard_workspace_bytes() bytes of device memory per rank, kept
 *                  between the calls of one step (no zeroing needed)
 *   send_k         this rank's message k, sc_shard_message_bytes(B, gamma, k) bytes
 *   gathered_k     the W messages k in rank order (W * sc_shard_message_bytes bytes)
 *   temperature    0 < T < inf (greedy decoding is sc_verify's)
 *   rule, alpha    SC_RULE_CHOW .. SC_RULE_NEVER_DEFER, 0 <= alpha <= 1
 * The calls of one step must see the same B, gamma, W, shard_begin, rule, alpha
 * and temperature on every rank.  Size limit: B (gamma + 1) max(32, slices) <=
 * 2^31 - 1, slices = ceil(shard width / 4096) (the kernels' grids).
 */
#ifndef SC_SHARD_H_
#define SC_SHARD_H_

#include <stddef.h>
#include <stdint.h>
#include <cuda_runtime_api.h>

#include "sc.h"

#ifdef __cplusplus
extern "C" {
#endif

#define SC_SHARD_MAX 16

/* Bytes of one rank's message k (1..5) for B sequences of gamma drafts
 * (independent of V and W; 0 for another k). */
size_t sc_shard_message_bytes(int B, int gamma, int message);

/* Device workspace of one rank holding a shard of `width` tokens. */
size_t sc_shard_workspace_bytes(int B, int gamma, int width, sc_dtype dtype);

int sc_shard_pass1(const void *draft_shard, const void *target_shard, sc_dtype dtype, int64_t ld,
                   const int32_t *draft_tokens, int B, int gamma, int W, int rank,
                   const int *shard_begin, float temperature, sc_rule rule, void *workspace,
                   size_t workspace_bytes, void *send1, cudaStream_t stream);

/* send2 is written only with SC_RULE_OPT (NULL is allowed otherwise). */
int sc_shard_decide(const void *draft_shard, const void *target_shard, sc_dtype dtype, int64_t ld,
                    const void *gathered1, const int32_t *draft_tokens, const float *uniforms,
                    int B, int gamma, int W, int rank, const int *shard_begin, sc_rule rule,
                    float alpha, float temperature, void *workspace, size_t workspace_bytes,
                    void *send2, int32_t *device_status, cudaStream_t stream);

/* SC_RULE_OPT only (another rule is SC_ERR_INVALID_ARG). */
int sc_shard_tv(const void *draft_shard, const void *target_shard, sc_dtype dtype, int64_t ld,
                const void *gathered2, int B, int gamma, int W, int rank, const int *shard_begin,
                sc_rule rule, float alpha, float temperature, void *workspace,
                size_t workspace_bytes, void *send3, cudaStream_t stream);

/* gathered3 is read only with SC_RULE_OPT (NULL is allowed otherwise). */
int sc_shard_accept(const void *draft_shard, const void *target_shard, sc_dtype dtype, int64_t ld,
                    const void *gathered3, const float *uniforms, int B, int gamma, int W,
                    int rank, const int *shard_begin, sc_rule rule, float alpha,
                    float temperature, void *workspace, size_t workspace_bytes, void *send4,
                    cudaStream_t stream);

int sc_shard_draw(const void *draft_shard, const void *target_shard, sc_dtype dtype, int64_t ld,
                  const void *gathered4, const float *uniforms, int B, int gamma, int W, int rank,
                  const int *shard_begin, float temperature, void *workspace,
                  size_t workspace_bytes, void *send5, cudaStream_t stream);

/* num_accepted [B] int32: j*; next_token [B] int32: the token emitted at j*. */
int sc_shard_finish(const void *gathered5, int B, int gamma, int W, const void *workspace,
                    size_t workspace_bytes, int32_t *num_accepted, int32_t *next_token,
                    cudaStream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* SC_SHARD_H_ */
