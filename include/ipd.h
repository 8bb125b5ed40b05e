/*
 * ipd.h -- C ABI of the IPD verify-step library (libipd.so, sm_103a).
 *
 * The verify step of Interactive-Policy Distillation's bidirectional
 * propose-and-verify rollout (Sec. 3.2.1 and the fused engine of Sec. 3.2.3):
 * the verifier scores the span of tokens the other model just proposed.
 *
 *   ipd_verify_attn  span-causal attention of the verifier's k span queries
 *                    over its own paged KV cache, co-launched with the
 *                    proposer's q_len = 1 decode attention over the other
 *                    model's cache (different GQA shapes, one launch).
 *   ipd_decode_attn  the decode attention alone.
 *   ipd_score_span   one pass over both models' logits of every span
 *                    position: log-softmax, per-token log-probs, the
 *                    teacher-feedback term, top-K coverage, union-support
 *                    top-K KL in both directions, the accept / takeover /
 *                    handback verdict and the new cache lengths.
 *   ipd_score_span_needed  the same verdict and loss inputs from only the
 *                    logits rows they need (the verifier's up to each
 *                    request's first transition, the proposer's at the
 *                    emitted positions).
 *   ipd_split_loss   the source-split objective of the step.
 *
 * Beyond the step itself: ipd_score_span_ex (other takeover / handback rules,
 * entropies, top-K overlap, top-K lists, the next span's first token),
 * ipd_full_kl (full-vocabulary KL both ways), ipd_sample (seeded sampling of
 * rows), ipd_kv_append / ipd_kv_append_many (new K/V rows into paged caches)
 * and ipd_split_loss_grad (the objective's gradient with respect to the
 * student's logits, sparse and dense).
 *
 * Conventions for every call
 *   - Data pointers are DEVICE pointers owned by the caller; the library never
 *     allocates.  Scratch memory comes from a caller-provided device workspace
 *     whose size the matching *_workspace_size query returns (host-only
 *     arithmetic; the queries never touch the GPU).
 *   - Every call is asynchronous on the caller's stream and never synchronises.
 *   - bf16 tensors are passed as uint16_t bit patterns.
 *   - Arguments are validated on the host before anything is launched; a
 *     failed check returns a status and launches nothing.  Conditions that
 *     only the device can see (a page id outside the pool, a length beyond
 *     the page table) are caught by the kernels, which skip the offending
 *     access and record a code readable with ipd_get_device_error().
 *   - Returns IPD_OK or one of the IPD_ERR_* codes below.
 */
#ifndef IPD_H_
#define IPD_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

struct CUstream_st;
typedef struct CUstream_st *ipd_stream_t; /* same handle as cudaStream_t */

#define IPD_OK 0
#define IPD_ERR_INVALID_ARG 1 /* null pointer, negative size, inconsistent shape */
#define IPD_ERR_UNSUPPORTED 2 /* head_dim != 128, page_size != 16, K > 32, ... */
#define IPD_ERR_WORKSPACE 3   /* workspace null or smaller than the query says */
#define IPD_ERR_CUDA 4        /* a CUDA runtime call failed (launch, attribute) */
#define IPD_ERR_TIMEOUT 5     /* a bounded device wait ran out (never expected) */
#define IPD_ERR_DEVICE 6      /* device-side check recorded an error */
#define IPD_ERR_CAPACITY 7    /* more work than a fixed-size entry point holds */

/* Device-side error codes (ipd_get_device_error). */
#define IPD_DEVERR_NONE 0u
#define IPD_DEVERR_PAGE_ID 1u    /* page_table entry < 0 or >= num_pages    */
#define IPD_DEVERR_SEQ_LEN 2u    /* seq_len < q_len or > max_pages*16, or q_len > max_q_len */
#define IPD_DEVERR_TOKEN 3u      /* proposed token id outside [0, vocab)     */
#define IPD_DEVERR_PLAN 4u       /* work list larger than the workspace     */
#define IPD_DEVERR_WAIT 5u       /* a bounded pipeline wait ran out         */
#define IPD_DEVERR_SPAN 6u       /* cu_span / cu_q / cu_new not non-decreasing, or rows past them */

#define IPD_MAX_BATCHES 8
#define IPD_MAX_K 32

/* One paged KV cache (one attention layer of one model).
 * k_pages, v_pages: [num_pages][num_kv_heads][page_size][head_dim] bf16,
 * row-major, 16-byte aligned.  A page holds page_size consecutive token
 * positions of every KV head (vLLM-style paging, Sec. 3.2.3).
 * Supported: page_size == 16, head_dim == 128, 1 <= num_kv_heads <= 64. */
typedef struct ipd_kv_cache {
  const uint16_t *k_pages;
  const uint16_t *v_pages;
  int64_t num_pages;
  int32_t page_size;
  int32_t num_kv_heads;
  int32_t head_dim;
} ipd_kv_cache;

/* A sub-batch of requests attending one cache.
 *  cache       host pointer to the cache descriptor.
 *  num_q_heads multiple of cache->num_kv_heads; query head h reads KV head
 *              h / (num_q_heads / num_kv_heads) (grouped-query attention).
 *  q           [total_q][num_q_heads][head_dim] bf16.
 *  cu_q        [num_reqs + 1] int32 prefix offsets into q; request r has
 *              q_len = cu_q[r+1] - cu_q[r] queries (the span length k_r for a
 *              verify batch, 1 for a decode batch).
 *  seq_len     [num_reqs] int32 KV length L_r in this cache, INCLUDING the
 *              span (whose K/V are already written at positions L_r-k_r..L_r-1).
 *              Query i of request r sits at position L_r - q_len + i and sees
 *              keys 0 .. L_r - q_len + i (causal within the span).
 *  page_table  [num_reqs][max_pages] int32; entry p of row r is the pool page
 *              holding positions 16p .. 16p+15 of request r.  Only the first
 *              ceil(L_r / 16) entries of a row are read.
 *  total_q, max_q_len, max_seq_len: host-known bounds (total_q must equal
 *              cu_q[num_reqs]); they size the grid and the workspace without
 *              a device-to-host read.
 *  out         [total_q][num_q_heads][head_dim] bf16, written by the call. */
typedef struct ipd_attn_batch {
  const ipd_kv_cache *cache;
  int32_t num_q_heads;
  int32_t num_reqs;
  const uint16_t *q;
  const int32_t *cu_q;
  const int32_t *seq_len;
  const int32_t *page_table;
  int32_t max_pages;
  int32_t total_q;
  int32_t max_q_len;
  int32_t max_seq_len;
  uint16_t *out;
} ipd_attn_batch;

/* Workspace bytes for one ipd_verify_attn / ipd_decode_attn call on these
 * batches (host arithmetic only).  Returns 0 if the batches are invalid. */
size_t ipd_attn_workspace_size(const ipd_attn_batch *verify, int n_verify,
                               const ipd_attn_batch *decode, int n_decode);

/* Span-verify attention (Sec. 3.2.3, verification stage: every verifier
 * prefills the unverified drafts of its sub-batch in one pass over its own
 * cache) for n_verify batches, together with the proposer decode attention
 * (proposal stage: each proposer extends only its own cache) for n_decode
 * batches, in ONE launch.  decode may be NULL when n_decode == 0.
 * n_verify + n_decode <= IPD_MAX_BATCHES.  softmax_scale is applied to q.k
 * (1/sqrt(head_dim) for the configurations of this library's tests).
 * out = softmax(scale * q K^T) V per query and head, fp32 accumulation,
 * rounded to bf16 once. */
int ipd_verify_attn(const ipd_attn_batch *verify, int n_verify,
                    const ipd_attn_batch *decode, int n_decode,
                    float softmax_scale, void *workspace, size_t workspace_bytes,
                    ipd_stream_t stream);

/* The decode attention alone (same semantics, q_len = 1 per request). */
int ipd_decode_attn(const ipd_attn_batch *decode, int n_decode, float softmax_scale,
                    void *workspace, size_t workspace_bytes, ipd_stream_t stream);

/* Workspace bytes for ipd_score_span. */
size_t ipd_score_workspace_size(int num_reqs, int total_tokens, int vocab, int K);

/* The vocabulary pass, verdict and cache bookkeeping of one verify step.
 *
 * Inputs
 *  logits_student [total_tokens][vocab] bf16: row t is the student's logits
 *                 pi(.|c_t) at span position t (flat over requests).
 *  logits_teacher [total_tokens][vocab] bf16: the teacher's q(.|c_t).
 *  tokens         [total_tokens] int32: the proposed token at each position.
 *  cu_span        [num_reqs + 1] int32 prefix offsets of each request's span.
 *  driver         [num_reqs] uint8: 0 = the student proposed (teacher
 *                 verifies), 1 = the teacher proposed (student verifies).
 *  prefix_len     [num_reqs] int32: verified prefix length before the span.
 *  K              top-K width, 1 <= K <= 32, K <= vocab (Sec. 4.1 uses 16).
 *  eos_id         end-of-sequence token id, or -1 for none.
 *
 * Per-token outputs [total_tokens]
 *  logp_s, logp_t full-vocabulary log-probabilities of the proposed token
 *                 under the student and the teacher.
 *  feedback       log q(x_t) - log pi(x_t): the per-token teacher-feedback
 *                 reward, minus the sampled-token estimate of Eq.
 *                 (sampled_token_opd).
 *  kl_rev         KL(pi_bar || q_bar) on S_t = Top_K(pi) u Top_K(q), both
 *                 renormalised on S_t (Eq. topk_normalization,
 *                 topk_opd_on_sequence); the on-policy term of Eq. ipd_off_loss.
 *  kl_fwd         KL(q_bar || pi_bar) on the same support; the off-policy term.
 *  covered        1 if the proposed token is in the VERIFIER's Top_K, else 0.
 *                 Top_K orders by logit, ties broken by smaller token id.
 *  margin         verifier logit of the proposed token minus the verifier's
 *                 K-th largest logit (0 on an exact tie at the boundary).
 *  source         0 = emitted with z = S, 1 = emitted with z = T, 255 = not
 *                 emitted (rejected or after the transition).
 * Per-request outputs [num_reqs]
 *  first_trans    first position whose verdict changes the driver (takeover
 *                 for driver 0, handback for driver 1), or k_r if none occurs
 *                 before the span ends or an accepted EOS.
 *  n_emit         tokens emitted by this step.
 *  next_driver    driver after the step.
 *  new_len        prefix_len + n_emit: the length both caches roll back to.
 *  done           1 if an accepted EOS ended the request.
 * The verdict follows Eq. (ipd_state_transition) and the verdict-stage rules
 * of Sec. 3.2.3: a rejected student token is not emitted (the teacher
 * regenerates it), a handback token is kept, a student EOS counts only when
 * covered, a teacher EOS is accepted directly. */
int ipd_score_span(const uint16_t *logits_student, const uint16_t *logits_teacher,
                   const int32_t *tokens, const int32_t *cu_span, const uint8_t *driver,
                   const int32_t *prefix_len, int num_reqs, int total_tokens, int vocab,
                   int K, int eos_id,
                   float *logp_s, float *logp_t, float *feedback, float *kl_rev,
                   float *kl_fwd, uint8_t *covered, float *margin, uint8_t *source,
                   int32_t *first_trans, int32_t *n_emit, uint8_t *next_driver,
                   int32_t *new_len, uint8_t *done,
                   void *workspace, size_t workspace_bytes, ipd_stream_t stream);

/* ipd_score_span reading only the logits rows the step needs: the verifier's
 * rows up to each request's first transition and the proposer's rows of the
 * emitted positions (Sec. 3.2.3: tokens after the transition are discarded,
 * so neither model's row there enters the verdict or the loss).  Rows past a
 * transition that is already known when their turn comes are not read; the
 * rest are read as by ipd_score_span, position 0 of every request first.
 * A call whose rows all fit one wave of row CTAs reads every row (no
 * transition is known before every row has started).
 *
 * Arguments as for ipd_score_span, plus
 *  max_span       an upper bound (1 .. 65535) on every request's span length;
 *                 a longer span records IPD_DEVERR_SPAN and leaves that
 *                 request's outputs undefined.
 * Outputs: first_trans, n_emit, next_driver, new_len, done and source as
 * ipd_score_span.  logp_s, logp_t, feedback, kl_rev and kl_fwd as
 * ipd_score_span at every emitted position (source != 255), covered and
 * margin at every position up to the request's first transition; at the other
 * positions each of these is either ipd_score_span's value or, where a row
 * was not read, NaN (covered 0).  Only the default (top-K) rules.  Workspace
 * as for ipd_score_span (ipd_score_workspace_size). */
int ipd_score_span_needed(const uint16_t *logits_student, const uint16_t *logits_teacher,
                          const int32_t *tokens, const int32_t *cu_span, const uint8_t *driver,
                          const int32_t *prefix_len, int num_reqs, int total_tokens, int vocab,
                          int K, int eos_id, int max_span,
                          float *logp_s, float *logp_t, float *feedback, float *kl_rev,
                          float *kl_fwd, uint8_t *covered, float *margin, uint8_t *source,
                          int32_t *first_trans, int32_t *n_emit, uint8_t *next_driver,
                          int32_t *new_len, uint8_t *done,
                          void *workspace, size_t workspace_bytes, ipd_stream_t stream);

/* Takeover / handback rules (Sec. 3.2.1: top-K coverage is IPD's rule, but the
 * framework admits others, possibly different for takeover and handback, for
 * example a threshold on the entropy of either model; SKD is top-K takeover
 * with a fixed one-token handback).  A rule is a per-position predicate:
 * under the takeover rule (student-proposed spans) true = accept the student
 * token, under the handback rule (teacher-proposed spans) true = hand back
 * after this teacher token. */
#define IPD_RULE_TOPK 0      /* the proposed token is in the verifier's Top_K */
#define IPD_RULE_ENTROPY_S 1 /* H(pi_t) <= tau (student's full-vocabulary entropy, nats) */
#define IPD_RULE_ENTROPY_T 2 /* H(q_t) <= tau (teacher's) */
#define IPD_RULE_ALWAYS 3    /* true: OPD as a takeover rule, SKD's handback */
#define IPD_RULE_NEVER 4     /* false: the teacher keeps driving, as a handback rule */

/* Options and optional outputs of ipd_score_span_ex. */
typedef struct {
  int takeover_rule;   /* IPD_RULE_*: governs spans with driver 0 */
  int handback_rule;   /* IPD_RULE_*: governs spans with driver 1 */
  float takeover_tau;  /* threshold of the entropy rules, nats */
  float handback_tau;
  float *entropy_s;    /* [total_tokens] H(pi_t) over the full vocabulary, or NULL */
  float *entropy_t;    /* [total_tokens] H(q_t), or NULL */
  float *topk_overlap; /* [total_tokens] |Top_K(pi_t) n Top_K(q_t)| / K (Sec. 4.2), or NULL */
  int32_t *topk_s;     /* [total_tokens][K] Top_K(pi_t) token ids, best first (ties: lower id
                          first), or NULL; ipd_split_loss_grad takes these lists */
  int32_t *topk_t;     /* [total_tokens][K] Top_K(q_t), same order, or NULL */
  int32_t *next_token; /* [num_reqs] first token of each request's next span, drawn (as
                          ipd_sample does) from the next driver's row n_emit[r] of the span
                          with draw number draw_base[r] + prefix_len[r] + n_emit[r]; -1 when
                          the request ended or every span token was emitted; or NULL */
  const uint64_t *draw_base; /* [num_reqs] device, or NULL for 0 */
  uint64_t sample_seed;
  float inv_temperature;     /* > 0 and finite when next_token is set (1 = the paper's rollouts) */
} ipd_score_ext;

/* ipd_score_span with selectable rules and by-products.  ext == NULL is the
 * default (top-K coverage both ways, no extra outputs) and is exactly
 * ipd_score_span.  With other rules, `covered` holds the governing rule's
 * predicate and `margin` its signed distance from the threshold (tau - H for
 * the entropy rules, +inf / -inf for ALWAYS / NEVER); the verdict applies
 * Eq. (ipd_state_transition) with that predicate in place of coverage.
 * Returns IPD_ERR_INVALID_ARG for an unknown rule or a NaN threshold. */
int ipd_score_span_ex(const uint16_t *logits_student, const uint16_t *logits_teacher,
                      const int32_t *tokens, const int32_t *cu_span, const uint8_t *driver,
                      const int32_t *prefix_len, int num_reqs, int total_tokens, int vocab,
                      int K, int eos_id,
                      float *logp_s, float *logp_t, float *feedback, float *kl_rev,
                      float *kl_fwd, uint8_t *covered, float *margin, uint8_t *source,
                      int32_t *first_trans, int32_t *n_emit, uint8_t *next_driver,
                      int32_t *new_len, uint8_t *done, const ipd_score_ext *ext,
                      void *workspace, size_t workspace_bytes, ipd_stream_t stream);

/* Full-vocabulary KL of Eq. (full_vocab_opd) at every span position, in both
 * directions: kl_rev_full[t] = KL(pi_t || q_t) = sum_v pi(v) (log pi(v) -
 * log q(v)) and kl_fwd_full[t] = KL(q_t || pi_t).  A by-product for
 * monitoring (the quantity top-K OPD approximates, Sec. 3.1); one read of both
 * logits rows per position.  logits_* as in ipd_score_span; outputs
 * [total_tokens] fp32 device arrays.  No workspace.  Returns
 * IPD_ERR_UNSUPPORTED unless vocab is a positive multiple of 8, and
 * IPD_ERR_INVALID_ARG for NULL or misaligned (16-byte) pointers. */
int ipd_full_kl(const uint16_t *logits_student, const uint16_t *logits_teacher,
                int total_tokens, int vocab, float *kl_rev_full, float *kl_fwd_full,
                ipd_stream_t stream);

/* ipd_score_span for callers that cannot allocate device memory.
 *
 * No counterpart in the paper: this is a calling convention of the library.
 * Some callers cannot hand the library a workspace: an operator plugged into
 * a runtime whose interface passes only inputs and outputs and which forbids
 * allocating inside the step, or a serving loop that must not call the
 * allocator because cudaMalloc / cudaFree can synchronise the device.  This
 * entry point takes no workspace and allocates nothing (no cudaMalloc, no
 * cudaFree, no allocating library routine).  Its scratch is one array in the
 * library's static device memory, sized for IPD_STATIC_MAX_TOKENS span
 * positions (about 2.1 MiB), which every GPU that loads the library holds
 * until the process exits.
 *
 * Arguments, outputs and semantics are those of ipd_score_span without the
 * workspace.  total_tokens > IPD_STATIC_MAX_TOKENS returns IPD_ERR_CAPACITY
 * and launches nothing.  The first call on a device looks up the array's
 * device address (cudaGetSymbolAddress, once per device, with that device
 * current); make that first call before any stream capture.  All calls share
 * the one array, so calls that overlap on the GPU (on different streams, or
 * from different host threads) race on it and their results are undefined:
 * serialise them.  The array keeps the last call's contents; nothing in it
 * needs to start at zero. */
#define IPD_STATIC_MAX_TOKENS 4096
int ipd_score_span_static(const uint16_t *logits_student, const uint16_t *logits_teacher,
                          const int32_t *tokens, const int32_t *cu_span, const uint8_t *driver,
                          const int32_t *prefix_len, int num_reqs, int total_tokens, int vocab,
                          int K, int eos_id,
                          float *logp_s, float *logp_t, float *feedback, float *kl_rev,
                          float *kl_fwd, uint8_t *covered, float *margin, uint8_t *source,
                          int32_t *first_trans, int32_t *n_emit, uint8_t *next_driver,
                          int32_t *new_len, uint8_t *done, ipd_stream_t stream);

/* Loss direction per token source (the KL-direction ablation of Sec. 4.3). */
#define IPD_DIR_SPLIT 0    /* z=S: KL(pi||q), z=T: KL(q||pi)   (IPD default) */
#define IPD_DIR_REVERSE 1  /* both reverse                                   */
#define IPD_DIR_FORWARD 2  /* both forward                                   */
#define IPD_DIR_INVERSE 3  /* z=S: forward, z=T: reverse                     */
/* Aggregation (Eq. ipd_objective and App. B.3). */
#define IPD_AGG_SEQ_MEAN_TOKEN_MEAN 0
#define IPD_AGG_GLOBAL_TOKEN_MEAN 1

/* Workspace bytes for ipd_split_loss (0: it needs none). */
size_t ipd_loss_workspace_size(int num_reqs);

/* The source-split objective of one step (Eq. ipd_off_loss, ipd_objective).
 *  kl_rev, kl_fwd, source, n_emit, cu_span: as produced by ipd_score_span.
 *  resp_len  [num_reqs] int32 response lengths |x_r| for the length
 *            normalisation, or NULL to use n_emit.  Requests whose length is
 *            0 are left out of the batch mean.
 *  out8      8 floats (device): loss, sum_on, sum_off, n_on, n_off,
 *            intervention_ratio (share of teacher-sourced tokens), numer,
 *            denom (loss = numer / denom, so shards of a batch can be
 *            combined by summing numer and denom).
 * The reduction order is fixed, so the result is bitwise reproducible. */
int ipd_split_loss(const float *kl_rev, const float *kl_fwd, const uint8_t *source,
                   const int32_t *cu_span, const int32_t *n_emit, const int32_t *resp_len,
                   int num_reqs, int agg_mode, int dir_mode, float *out8,
                   void *workspace, size_t workspace_bytes, ipd_stream_t stream);

/* Writes the K/V rows of newly computed tokens into a paged cache (Sec. 3.2.3:
 * the proposer's decode extends its own cache by one token, the verifier's
 * prefill writes the span's k tokens into its cache; each before the
 * attention that reads them).
 *  k_pages, v_pages  [num_pages][num_kv_heads][16][128] bf16, written in place
 *  k_new, v_new      [total_new][num_kv_heads][128] bf16 rows of the new tokens
 *  cu_new            [num_reqs + 1] int32: request r owns rows cu_new[r] .. cu_new[r+1]-1
 *  seq_len           [num_reqs] int32 sequence length AFTER the append: row i of
 *                    request r (n_r rows) goes to position seq_len[r] - n_r + i,
 *                    page page_table[r][pos / 16], slot pos % 16
 *  page_table        [num_reqs][max_pages] int32, as in ipd_attn_batch
 * All pointers 16-byte aligned.  Returns IPD_ERR_UNSUPPORTED unless
 * page_size == 16 and head_dim == 128.  A row outside cu_new[0] ..
 * cu_new[num_reqs] - 1 (IPD_DEVERR_SPAN), a position outside the page table
 * or at or past seq_len (IPD_DEVERR_SEQ_LEN) and a page id outside the pool
 * (IPD_DEVERR_PAGE_ID) are recorded and that row is skipped.  Rolling a cache back after a
 * verdict needs no kernel: the next step passes the shorter length. */
int ipd_kv_append(uint16_t *k_pages, uint16_t *v_pages, int64_t num_pages, int num_kv_heads,
                  int page_size, int head_dim, const uint16_t *k_new, const uint16_t *v_new,
                  const int32_t *cu_new, const int32_t *seq_len, const int32_t *page_table,
                  int max_pages, int num_reqs, int total_new, ipd_stream_t stream);

/* One append of ipd_kv_append_many: the arguments of ipd_kv_append. */
typedef struct {
  uint16_t *k_pages, *v_pages;
  int64_t num_pages;
  int num_kv_heads, page_size, head_dim;
  const uint16_t *k_new, *v_new;
  const int32_t *cu_new, *seq_len, *page_table;
  int max_pages, num_reqs, total_new;
} ipd_kv_append_desc;

/* Several appends (a step's span rows into each verifier's cache and decode
 * rows into each proposer's cache) in one launch: appends[0 .. n-1], n <=
 * IPD_MAX_BATCHES, each with the meaning, checks and device error behaviour
 * of ipd_kv_append.  The descriptor array is host memory, read during the
 * call.  Any invalid descriptor returns its error and launches nothing.  Two
 * appends must not write the same page slot. */
int ipd_kv_append_many(const ipd_kv_append_desc *appends, int n, ipd_stream_t stream);

/* Seeded sampling from softmax(l * inv_temperature) of each row (training
 * rollouts sample at temperature 1, top-p 1: App. A).  A draw is a fixed
 * function of (row, seed, draw number, inv_temperature), reproducible on any
 * device:
 *   bits_v = word v % 4 of Philox4x32-10(counter (v / 4, draw_lo, draw_hi, 0),
 *            key (seed_lo, seed_hi))  (Salmon et al., SC 2011)
 *   u_v    = (2 (bits_v >> 9) + 1) * 2^-24
 *   s_v    = fl(l_v * c) - lg2(-lg2(u_v)),  c = fl(fp32(log2 e) * inv_temperature)
 *   token  = argmax_v s_v (ties to the lower id)
 * where every product and sum is rounded to fp32 separately and lg2(x), for
 * x = 2^e m with m in (sqrt(1/2), sqrt(2)], is e + t P(t), t = m - 1, P by
 * Horner's rule with the fp32 coefficients (bit patterns, lowest degree first)
 * 3FB8AA3A BF38AA93 3EF63BAD BEB871A3 3E92FB93 BE7ECB25 3E6FD4B5 BE15B661.
 * This is the Gumbel-max trick in base 2, so the token follows
 * softmax(l * inv_temperature).
 *  logits   [n_rows][vocab] bf16, 16-byte aligned, vocab a multiple of 8
 *  draw_id  [n_rows] uint64 draw numbers (device), or NULL for all 0
 *  tokens   [n_rows] int32 output
 * Returns IPD_ERR_INVALID_ARG for a non-positive or non-finite
 * inv_temperature or a missing pointer, IPD_ERR_UNSUPPORTED for vocab % 8 != 0,
 * IPD_ERR_WORKSPACE for a workspace below ipd_sample_workspace_size. */
size_t ipd_sample_workspace_size(int n_rows, int vocab);
int ipd_sample(const uint16_t *logits, int n_rows, int vocab, uint64_t seed,
               const uint64_t *draw_id, float inv_temperature, int32_t *tokens, void *workspace,
               size_t workspace_bytes, ipd_stream_t stream);

/* Element type of the dense gradient of ipd_split_loss_grad. */
#define IPD_DTYPE_F32 0
#define IPD_DTYPE_BF16 1

/* Workspace bytes for ipd_split_loss_grad (0: it needs none). */
size_t ipd_loss_grad_workspace_size(int total_tokens, int K);

/* Gradient of grad_scale * loss with respect to the student's logits, for the
 * loss of ipd_split_loss (Eq. ipd_off_loss and Eq. ipd_objective; top-K
 * renormalisation of Eq. topk_normalization).  The supports
 * S_t = Top_K(pi_t) u Top_K(q_t) are piecewise constant in the logits and are
 * held fixed.  Position t, when emitted, carries weight w_t = 1 / (D |x_r|)
 * (agg_mode 0, D = number of requests with |x_r| > 0) or 1 / D (agg_mode 1,
 * D = sum of those |x_r|); D is read from loss_out8[7], the `denom` output of
 * ipd_split_loss, so a sharded batch passes its combined denominator.  With
 * pi_bar, q_bar the two softmaxes restricted to S_t, for v in S_t:
 *   reverse KL(pi_bar || q_bar): w_t pi_bar_v (log pi_bar_v - log q_bar_v - KL)
 *   forward KL(q_bar || pi_bar): w_t (pi_bar_v - q_bar_v)
 * (the direction per source as in ipd_split_loss's dir_mode); every other
 * logit, and every position that was not emitted, has gradient 0.
 *  logits_student, logits_teacher  [total_tokens][vocab] bf16 (as for ipd_score_span)
 *  topk_s, topk_t  [total_tokens][K] int32, the lists ipd_score_span_ex writes
 *  source, cu_span, n_emit, resp_len, num_reqs, agg_mode, dir_mode  as for ipd_split_loss
 *  loss_out8       the 8 floats ipd_split_loss wrote (device)
 *  grad_idx, grad_val  [total_tokens][2K] sparse gradient (required): slots
 *      0..K-1 hold Top_K(pi_t) in order, slots K..2K-1 the entries of
 *      Top_K(q_t) not in Top_K(pi_t); unused slots and positions with no
 *      gradient hold id -1 and value 0
 *  grad_dense      [total_tokens][vocab] dense gradient of dense_dtype
 *      (IPD_DTYPE_F32 or IPD_DTYPE_BF16, round to nearest even), 16-byte
 *      aligned, or NULL for the sparse form only
 * Returns IPD_ERR_INVALID_ARG for a missing pointer, an unknown mode or dtype,
 * a non-finite grad_scale or a misaligned grad_dense; IPD_ERR_UNSUPPORTED for
 * K outside [1, IPD_MAX_K] or K > vocab.  An id outside [0, vocab) in the
 * top-K lists is recorded as IPD_DEVERR_TOKEN and that position gets no
 * gradient. */
int ipd_split_loss_grad(const uint16_t *logits_student, const uint16_t *logits_teacher,
                        const int32_t *topk_s, const int32_t *topk_t, const uint8_t *source,
                        const int32_t *cu_span, const int32_t *n_emit, const int32_t *resp_len,
                        const float *loss_out8, int num_reqs, int total_tokens, int vocab, int K,
                        int agg_mode, int dir_mode, float grad_scale, int32_t *grad_idx,
                        float *grad_val, void *grad_dense, int dense_dtype, void *workspace,
                        size_t workspace_bytes, ipd_stream_t stream);

/* Measurement aid.  While on, every ipd_verify_attn / ipd_decode_attn call
 * records CUDA events on its stream around its attention kernel alone (not
 * the planner), for up to 4096 calls; ipd_attn_kernel_time synchronises on
 * them, returns the summed kernel time and the number of timed launches, and
 * starts a new record.  Not for use while capturing a CUDA graph, nor from
 * several host threads at once. */
int ipd_set_attn_kernel_timing(int on);
int ipd_attn_kernel_time(double *total_ms, int *launches);

/* Reads and clears the device error word of the current device
 * (synchronises the device).  *code receives an IPD_DEVERR_* value. */
int ipd_get_device_error(uint32_t *code);

/* Human-readable name of a status code (static storage). */
const char *ipd_status_string(int status);

/* Library version, e.g. 100 for 0.1.0. */
int ipd_version(void);

/* Whether the current device's kernels can read `ptr` at that same address:
 * device memory of the current device, managed memory, or page-locked host
 * memory mapped into the device's address space (cudaHostAlloc under unified
 * addressing).  *readable = 1 or 0; a pointer CUDA does not know is 0.  Lets
 * a caller hand host-resident inputs (for example logits rows) to the calls
 * directly, so that only the bytes a kernel reads cross the host link. */
int ipd_device_readable(const void *ptr, int *readable);

#ifdef __cplusplus
}
#endif
#endif /* IPD_H_ */
