/*
 * spo.h -- C ABI of libspo: the GRPO policy log-prob / policy-loss hot path of
 * CUDAPerf (arxiv 2607.20908) on NVIDIA GB300 (sm_103a).
 *
 * The paper's online RL phase (section 3, "Multi-turn RL Training") maximises
 * the GRPO objective of Eq. 3: for every rollout token it needs the policy's
 * log-probability of the sampled token over the full vocabulary, the ratio
 * against the old policy, group-normalised advantages of the composite reward,
 * the clipped surrogate with a KL term, and the gradient of all of it back to
 * the final hidden states H and the LM-head weight W.  This header is that
 * path, one call per step:
 *
 *   spo_token_select       loss tokens: mask, ignore index, 1024-token window
 *   spo_logprobs_fwd       logits H W^T tile by tile + online logsumexp
 *                          (logits never reach memory) -> logp, entropy, lse
 *   spo_group_advantages   A_hat_i = (r_i - mean_g) / (std_g + eps)
 *   spo_policy_loss_fwd    ratio, clip, KL, aggregation -> loss, dL/dlogp
 *   spo_policy_loss_bwd    dH = G W, dW = G^T H with
 *                          G = tau^-1 g (onehot - softmax), logits recomputed
 *
 * or all of it as one call, spo_grpo_step, with one workspace
 * (spo_workspace_size).  spo_policy_loss_bwd_ex adds hooks for overlapping the
 * multi-GPU exchanges (dW per vocabulary block, dH) with the GEMMs that follow.
 *
 * Conventions shared by every call
 *   - Every array argument is a DEVICE pointer owned by the caller unless the
 *     comment says otherwise.  The library never allocates device memory,
 *     never frees, and never synchronises the stream (except
 *     spo_device_error and spo_sync_check, which say so).  Scratch memory
 *     comes only from the caller's `ws` buffer, sized by the matching
 *     *_workspace_size call (spo_policy_loss_fwd_noalloc, which has none,
 *     says where its scratch lives).
 *   - `stream` is a cudaStream_t (NULL = legacy default stream).  Work is
 *     enqueued asynchronously in stream order.  Calls on distinct workspaces
 *     may run concurrently on different streams.
 *   - Layouts are row-major and dense.  bf16 matrices (H, W, dH) must start on
 *     a 16-byte boundary (the tensor-memory-accelerator loads require it).
 *   - Argument errors are detected on the host before anything is enqueued
 *     and have no side effects; the status says which class of error, and
 *     spo_last_error() returns a one-line description (per host thread).
 *   - A launch failure returns SPO_ERR_CUDA.  Every device-side wait in the
 *     tensor-core kernels is bounded; a wait that expires records a code that
 *     spo_device_error() returns (SPO_ERR_TIMEOUT) instead of hanging.
 *   - Results are bit-reproducible run to run: every output element is
 *     reduced in one fixed order whatever the order in which tiles are
 *     scheduled.  The compute calls make no host synchronisation and no
 *     allocation, so a sequence of them can be captured into a CUDA graph
 *     (workspaces and buffers fixed) and replayed.
 *   - The sign convention is that of an optimiser: `loss` = -J_GRPO, to be
 *     minimised.
 *
 * Symbols: the precision of every result is stated per call.  Token ids are
 * already shifted (tgt[t] is the token whose probability row t predicts);
 * tgt[t] < 0 marks an ignored token (e.g. -100).
 */
#ifndef SPO_H_
#define SPO_H_

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define SPO_API __attribute__((visibility("default")))
#else
#define SPO_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum spo_status {
    SPO_OK = 0,
    SPO_ERR_INVALID_ARG = 1, /* null pointer, bad enum, non-finite scalar */
    SPO_ERR_SHAPE = 2,       /* sizes out of range or inconsistent         */
    SPO_ERR_ALIGNMENT = 3,   /* pointer or leading dimension misaligned    */
    SPO_ERR_WORKSPACE = 4,   /* ws NULL or smaller than *_workspace_size   */
    SPO_ERR_UNSUPPORTED = 5, /* device is not sm_103 / sm_100 class        */
    SPO_ERR_CUDA = 6,        /* a CUDA runtime call or launch failed       */
    SPO_ERR_TIMEOUT = 7      /* a bounded device wait expired              */
} spo_status;

/* Aggregation of per-token terms into the scalar objective (Eq. 3). */
typedef enum spo_agg {
    SPO_AGG_SEQ_GROUP = 0, /* Eq. 3: mean over groups of (1/G) sum_i (1/|o_i|) sum_t */
    SPO_AGG_TOKEN = 1      /* one mean over every loss token of the batch          */
} spo_agg;

/* Standard deviation used by the group-normalised advantage. */
typedef enum spo_std {
    SPO_STD_UNBIASED = 0,  /* divide the sum of squares by n - 1 */
    SPO_STD_POPULATION = 1 /* divide by n                        */
} spo_std;

/* Library version, (major << 16) | minor. */
SPO_API int spo_version(void);

/* Static text for a status code (never NULL). */
SPO_API const char* spo_status_string(int status);

/* Copies the calling host thread's description of its last failed call into
 * buf (NUL-terminated, truncated to n bytes).  Returns the status of that
 * call (SPO_OK if none failed). */
SPO_API int spo_last_error(char* buf, size_t n);

/* The same as spo_last_error, under the name and return type of the
 * boundary's specification: the calling thread's one-line description of its
 * last failed call, and that call's status. */
SPO_API spo_status spo_last_error_detail(char* buf, size_t n);

/* Reads and clears the device-side error word that bounded waits set on
 * timeout.  SYNCHRONISES `stream`.  *code receives 0 or the kernel's code.
 * Returns SPO_ERR_TIMEOUT if a wait expired, else SPO_OK / SPO_ERR_CUDA. */
SPO_API spo_status spo_device_error(int* code, void* stream);

/* spo_device_error without the code: SYNCHRONISES `stream`, then returns
 * SPO_ERR_CUDA if the stream's work failed, SPO_ERR_TIMEOUT if a bounded
 * device wait expired since the last check (clearing it), else SPO_OK. */
SPO_API spo_status spo_sync_check(void* stream);

/* Failure-detection self-test: enqueues one thread that waits, through the
 * tensor-core kernels' own bounded wait, on a shared-memory barrier nothing
 * ever arrives on.  The wait gives up after its limit (1 s), records code
 * 0x1ff in the error word and the kernel returns, so the context stays
 * usable; the next spo_device_error reports SPO_ERR_TIMEOUT with that code.
 * Faults, traps and hangs nothing. */
SPO_API spo_status spo_selftest_bounded_wait(void* stream);

/* ---------------------------------------------------------------------------
 * a1. Loss-token selection (section 3, "Multi-turn RL Training": the loss uses
 * only unmasked tokens within a 1024-token window of each generation).
 *
 * Sequence i (one generated output o_i, or one turn of it) spans tokens
 * [cu_seqlens[i], cu_seqlens[i+1]).  Token t of sequence i is a loss token
 * when mask[t] == 1, tgt[t] >= 0, and fewer than `window` earlier tokens of the
 * same sequence are loss tokens (window <= 0: no cap).
 *
 *   cu_seqlens int32[n_seq+1]  non-decreasing, cu[0] = 0, cu[n_seq] = T
 *   mask       uint8[T]        1 = generated token, 0 = prompt/feedback; NULL = all 1
 *   tgt        int32[T]
 *   loss_mask  uint8[T]  out   1 for loss tokens, else 0
 *   n_tok      int32[n_seq] out number of loss tokens of each sequence (|o_i|)
 * 1 <= n_seq <= 2^24, 1 <= T <= 2^30.  Bit-exact (integer work).  cu_seqlens
 * monotonicity is the caller's contract (device data is not inspected on the
 * host).
 * ------------------------------------------------------------------------- */
SPO_API spo_status spo_token_select(const int32_t* cu_seqlens, const uint8_t* mask,
                                    const int32_t* tgt, int32_t n_seq, int64_t T, int32_t window,
                                    uint8_t* loss_mask, int32_t* n_tok, void* stream);

/* ---------------------------------------------------------------------------
 * a2 + a3. Per-token policy log-probabilities over the full vocabulary: the
 * pi_theta(o_{i,t} | q, o_{i,<t}) in the ratio of Eq. 3.
 *
 *   z_t      = inv_temp * H[t] . W^T           (bf16 inputs, fp32 accumulate)
 *   lse_t    = log sum_v exp(z_t[v])
 *   logp[t]  = z_t[tgt[t]] - lse_t             (<= 0)
 *   entropy[t] = lse_t - sum_v softmax(z_t)[v] z_t[v]   (natural log)
 *
 * The T x V logits are produced tile by tile in tensor memory and reduced by
 * an online max / sum-exp epilogue; only per-(token, vocab-tile) partials and
 * the three per-token results reach device memory.
 *
 *   H        bf16[T, d]  row-major, 16-byte aligned
 *   W        bf16[V, d]  row-major (LM-head layout), 16-byte aligned
 *   tgt      int32[T]    values in [0, V) for kept tokens (not range-checked)
 *   mask     uint8[T]    tokens with mask[t] == 0 are skipped; NULL = keep all
 *   sizes    1 <= T <= 2^24, 64 <= d <= 65536 with d % 64 == 0,
 *            256 <= V <= 2^24 with V % 8 == 0
 *   logp, entropy, lse  fp32[T] out; skipped tokens (mask 0 or tgt < 0) get 0.
 *            entropy and lse may be NULL.  lse feeds spo_policy_loss_bwd.
 *   ws       device scratch of at least spo_logprobs_workspace_size bytes,
 *            256-byte aligned
 * Accuracy vs an fp64 evaluation on the same bf16 inputs: |d logp| and
 * |d entropy| are O(1e-5) for d ~ 5e3 (fp32 accumulation and exp2).
 * ------------------------------------------------------------------------- */
SPO_API spo_status spo_logprobs_workspace_size(int64_t T, int64_t d, int64_t V, size_t* bytes);
SPO_API spo_status spo_logprobs_fwd(const void* H, const void* W, const int32_t* tgt,
                                    const uint8_t* mask, int64_t T, int64_t d, int64_t V,
                                    float inv_temp, float* logp, float* entropy, float* lse,
                                    void* ws, size_t ws_bytes, void* stream);

/* ---------------------------------------------------------------------------
 * Composite reward (section 2.2, "Verifiable Reward"; r_i = R_ver(i) + R_str(i),
 * section 3), the input of spo_group_advantages.  Per candidate i:
 *   R_comp  = -alpha_comp                        if the program does not compile
 *   R_corr  = -alpha_wrong * (1 - p)             p = fraction of tests passed
 *   R_speed = alpha_speed * clip(log2 S, s_min, s_max)
 *   R_cv    = -alpha_cv * cv
 *   R_ver   = R_comp (not compiled) | R_corr (p < 1) | R_corr + R_speed + R_cv (p = 1)
 *   r       = R_ver + r_struct
 *
 *   compiled  uint8[n]   0 = compilation failed
 *   pass_rate fp32[n]    in [0, 1]
 *   speedup   fp32[n]    sequential / CUDA runtime; a value that is not > 0
 *                        counts as the lower clip bound
 *   cv        fp32[n]    coefficient of variation of the CUDA runtime
 *   r_struct  fp32[n]    structural score R_str, or NULL for 0
 *   params    HOST pointer, or NULL for the paper's values (3.0, 2.0, 1.0,
 *             0.5, -0.5, 4.0); must be finite with s_min <= s_max
 *   rewards   fp32[n] out.  fp32 arithmetic (log2f); within 1e-6 of fp64.
 * ------------------------------------------------------------------------- */
typedef struct spo_reward_params {
    float alpha_comp, alpha_wrong, alpha_speed, alpha_cv, s_min, s_max;
} spo_reward_params;
SPO_API spo_status spo_reward_compose(const uint8_t* compiled, const float* pass_rate,
                                      const float* speedup, const float* cv,
                                      const float* r_struct, int32_t n,
                                      const spo_reward_params* params, float* rewards,
                                      void* stream);

/* ---------------------------------------------------------------------------
 * Offline structural ranker (section 2.1, "Structural Reward"; architecture in
 * the appendix "MLP Ranker Architecture").  Features phi (11 per program:
 * coalescing, arithmetic intensity, occupancy, divergence, transfer,
 * atomics, syncthreads, kernels, threads per block, global accesses, ops)
 * are z-scored with the training split's mean and std, phi_hat = (phi - mu) /
 * sigma, and scored by s_psi: 11 -> 64 -> 32 -> 1 with ReLU.  The score is
 * the structural reward R_str.  Training minimises the pairwise logistic
 * ranking loss L = mean_k softplus(-(s(y+_k) - s(y-_k))).
 *
 * params: fp32[2881] packed row-major: W1[64][11], b1[64], W2[32][64], b2[32],
 *         w3[32], b3.  phi fp32[n][11]; mu, sigma fp32[11].
 * spo_ranker_scores: scores fp32[n] = s_psi(phi_hat) (inference, no dropout).
 * spo_ranker_pair_loss: pos / neg int32[n_pairs] row indices into phi (the
 *   y+ and y- of each pair; valid rows of phi, not range-checked); keep1
 *   uint8[n_pairs][2][64] / keep2 uint8[n_pairs][2][32] are optional dropout
 *   keep flags of the two hidden layers ([k][0] = y+, [k][1] = y-), kept
 *   units scaled by 1 / (1 - drop_p) (NULL = no dropout); loss fp32[1]; grad
 *   fp32[2881] = dL/dparams (may be NULL).  One warp per pair; gradients are
 *   summed in a fixed order (run-to-run deterministic).  fp32 arithmetic.
 *   ws >= spo_ranker_workspace_size(n_pairs) bytes, 256-byte aligned.
 * ------------------------------------------------------------------------- */
#define SPO_RANKER_FEATURES 11
#define SPO_RANKER_PARAMS 2881
SPO_API spo_status spo_ranker_scores(const float* phi, const float* mu, const float* sigma,
                                     int32_t n, const float* params, float* scores, void* stream);
SPO_API spo_status spo_ranker_workspace_size(int32_t n_pairs, size_t* bytes);
SPO_API spo_status spo_ranker_pair_loss(const float* phi, const float* mu, const float* sigma,
                                        const int32_t* pos, const int32_t* neg, int32_t n_pairs,
                                        const float* params, const uint8_t* keep1,
                                        const uint8_t* keep2, float drop_p, float* loss,
                                        float* grad, void* ws, size_t ws_bytes, void* stream);

/* ---------------------------------------------------------------------------
 * Content checks of device inputs that the other calls take on trust (the
 * host cannot read device data without a synchronisation).  Enqueues one
 * pass and writes counts (DEVICE int32[6], zeroed first) of:
 *   [0] tokens with tgt[t] >= V (tgt < 0 is the valid "ignore" marker)
 *   [1] violations of cu_seqlens: decreasing steps, cu[0] != 0, cu[n_seq] != T
 *   [2] group ids outside [0, n_groups)
 *   [3] non-finite rewards
 *   [4] non-finite old / reference log-probs
 *   [5] mask bytes other than 0 and 1
 * Every array pointer may be NULL to skip its checks.  All zero = valid.
 * ------------------------------------------------------------------------- */
SPO_API spo_status spo_validate_inputs(const int32_t* tgt, int64_t T, int64_t V,
                                       const int32_t* cu_seqlens, int32_t n_seq,
                                       const int32_t* group_id, int32_t n_groups,
                                       const float* rewards, const float* old_logp,
                                       const float* ref_logp, const uint8_t* mask,
                                       int32_t* counts, void* stream);

/* ---------------------------------------------------------------------------
 * x[i] *= alpha for i < n (alpha_dev: device fp32 scalar used instead of alpha
 * when non-NULL).  Used by the data-parallel step to weight a rank's loss and
 * dL/dlogp by its share of the global normaliser of Eq. 3's average.  Any
 * 4-byte-aligned x; n == 0 is a no-op (x may then be NULL).
 * ------------------------------------------------------------------------- */
SPO_API spo_status spo_scale_f32(float* x, int64_t n, float alpha, const float* alpha_dev,
                                 void* stream);

/* x[i] *= (float)(num[0] / den[0]) for i < n, or x[i] = 0 when den[0] == 0;
 * num and den are DEVICE fp64 scalars.  A data-parallel rank's weight in Eq.
 * 3's global average is its own count over the all-reduced count (groups for
 * SEQ_GROUP, loss tokens for TOKEN): this applies that weight without the
 * host reading either count.  n == 0 is a no-op (x may then be NULL). */
SPO_API spo_status spo_scale_f32_ratio(float* x, int64_t n, const double* num, const double* den,
                                       void* stream);

/* ---------------------------------------------------------------------------
 * a4. Group-normalised advantage (definition under Eq. 3):
 *   A_hat_i = (r_i - mean(r_g)) / (std(r_g) + eps), g = group_id[i].
 * Members of a group are taken in ascending i; the arithmetic is IEEE fp32
 * in one fixed order (sum, divide, sum of rounded squared deviations,
 * divide, sqrt, add eps, divide; no fused multiply-add), so results are
 * reproducible bit for bit.  Groups of size <= 1 or with all rewards equal
 * give exactly 0.
 *
 *   rewards  fp32[n_seq]   composite reward r_i = R_ver(i) + R_str(i)
 *   group_id int32[n_seq]  values in [0, n_groups); members need not be contiguous
 *   adv      fp32[n_seq] out
 * ------------------------------------------------------------------------- */
SPO_API spo_status spo_group_advantages(const float* rewards, const int32_t* group_id,
                                        int32_t n_seq, int32_t n_groups, int std_mode, float eps,
                                        float* adv, void* stream);

/* spo_group_advantages_ws: the same advantages, bit for bit, in
 * O(n_seq + n_groups) work when each group's sequences are contiguous (one
 * run of equal group ids, the usual packing of rollouts), for batches far
 * beyond one step's few hundred sequences.  When the ids are non-decreasing
 * one pass over ids and rewards does the whole job; otherwise a pass finds
 * each group's run, and if some group has more than one run the call falls
 * back to the per-group scan of spo_group_advantages.  Arguments as there, plus
 *   ws  >= spo_group_advantages_workspace_size(n_seq, n_groups) bytes,
 *       256-byte aligned (3 ints per group + 2).
 * Sequences whose group id lies outside [0, n_groups) get no advantage
 * written, as in spo_group_advantages. */
SPO_API spo_status spo_group_advantages_workspace_size(int32_t n_seq, int32_t n_groups,
                                                       size_t* bytes);
SPO_API spo_status spo_group_advantages_ws(const float* rewards, const int32_t* group_id,
                                           int32_t n_seq, int32_t n_groups, int std_mode,
                                           float eps, float* adv, void* ws, size_t ws_bytes,
                                           void* stream);

/* ---------------------------------------------------------------------------
 * a5. Clipped surrogate, KL and aggregation of Eq. 3, forward, plus
 * g[t] = dL/dlogp[t] for the backward.  Per loss token t of sequence i:
 *   rho  = exp(logp - old_logp)
 *   surr = min(rho A_i, clip(rho, 1 - clip_eps, 1 + clip_eps) A_i)
 *   kl   = exp(ref - logp) - (ref - logp) - 1       (k3 estimator)
 *   l_t  = -(surr - kl_beta * kl)
 *   loss = sum_t c_t l_t,  c_t = 1/(N_g |S_g| n_i) (SEQ_GROUP: N_g non-empty
 *          groups, |S_g| sequences in i's group, n_i loss tokens of i) or
 *          1/sum_i n_i (TOKEN).
 *   g[t] = c_t (-A_i rho [clip not binding] + kl_beta (1 - exp(ref - logp)));
 *          the clip binds when A_i > 0 and rho > 1 + eps, or A_i < 0 and
 *          rho < 1 - eps (the bound itself counts as not binding).
 *
 *   logp, old_logp fp32[T]; ref_logp fp32[T] or NULL (NULL or kl_beta == 0: no KL)
 *   adv        fp32[n_seq]  per-sequence advantage (broadcast to its tokens)
 *   cu_seqlens int32[n_seq+1], group_id int32[n_seq] in [0, n_groups)
 *   loss_mask  uint8[T]  (spo_token_select output)
 *   loss       fp32[1] out;  g fp32[T] out (0 off the loss set)
 *   stats      fp32[4] out or NULL: {clip fraction, mean ratio, mean kl,
 *              number of loss tokens} over loss tokens
 *   ws         >= spo_policy_loss_workspace_size bytes
 *   1 <= n_seq, n_groups <= 2^24, 1 <= T <= 2^30
 * The reduction order is fixed: a group of lanes per sequence (16 when the
 * sequences average at most 128 tokens, else 32) sums its tokens in fp32
 * (each lane its own tokens in order, then a fixed butterfly); the sums over
 * sequences run in two fixed stages whose split depends only on n_seq -- the
 * loss as an unevaluated pair of floats added with TwoSum (about 48
 * significant bits, so cancellation between groups costs no accuracy), the
 * ratio and KL statistics in fp32, the counts as integers -- so results are
 * deterministic run to run and across devices.
 * ------------------------------------------------------------------------- */
SPO_API spo_status spo_policy_loss_workspace_size(int32_t n_seq, int32_t n_groups, size_t* bytes);
SPO_API spo_status spo_policy_loss_fwd(const float* logp, const float* old_logp,
                                       const float* ref_logp, const float* adv,
                                       const int32_t* cu_seqlens, const int32_t* group_id,
                                       int32_t n_seq, int32_t n_groups, const uint8_t* loss_mask,
                                       int64_t T, float clip_eps, float kl_beta, int agg,
                                       float* loss, float* g, float* stats, void* ws,
                                       size_t ws_bytes, void* stream);

/* ---------------------------------------------------------------------------
 * a6 - a8. Backward of the loss through the log-probabilities to H and W (the
 * policy update that maximises Eq. 3):
 *   G[t, v] = inv_temp * g[t] * (1[v == tgt[t]] - exp(z_t[v] - lse[t]))
 *   dH      = G W        (bf16 out, fp32 accumulate)
 *   dW      = G^T H      (fp32 out, fp32 accumulate; += if accumulate_dW)
 * z is recomputed tile by tile with the tensor cores; G is staged in bf16
 * scratch (chunks of at most 32768 rows).  Rows with g[t] == 0 contribute
 * nothing and are skipped; their dH rows are written as 0.
 *
 *   H, W, tgt, T, d, V, inv_temp  as in spo_logprobs_fwd
 *   lse      fp32[T]   from spo_logprobs_fwd
 *   g        fp32[T]   from spo_policy_loss_fwd
 *   dH       bf16[T, d] out (may be NULL to skip it)
 *   dW       fp32[V, d] out (may be NULL to skip it)
 *   ws       >= spo_policy_loss_bwd_workspace_size bytes
 * Accuracy vs fp64 on the same inputs: relative L2 error O(1e-3) (bf16 G).
 * ------------------------------------------------------------------------- */
SPO_API spo_status spo_policy_loss_bwd_workspace_size(int64_t T, int64_t d, int64_t V,
                                                      size_t* bytes);
SPO_API spo_status spo_policy_loss_bwd(const void* H, const void* W, const int32_t* tgt,
                                       const float* lse, const float* g, int64_t T, int64_t d,
                                       int64_t V, float inv_temp, void* dH, float* dW,
                                       int accumulate_dW, void* ws, size_t ws_bytes, void* stream);

/* ---------------------------------------------------------------------------
 * The backward with hooks for overlapping its results' collectives (no
 * counterpart in the paper, which trains on two GPUs without describing how
 * gradients are exchanged).  In data-parallel training dW is summed over the
 * ranks; in the vocabulary split dH is.  With hooks, dW is computed in
 * n_dw_blocks contiguous blocks of vocabulary rows, and a caller's CUDA event
 * is recorded on `stream` as soon as every dH row is final (dh_event) and as
 * soon as each dW block is final (dw_block_events[k]), so a collective issued
 * on another stream after waiting on that event runs while the remaining
 * GEMMs do.  The GEMMs that follow the first event leave reserve_sms SMs of
 * the device free for such a collective's kernels (0: use every SM).
 *
 *   n_dw_blocks      >= 1; block k covers dW rows [s_k, s_{k+1}) from
 *                    spo_dw_block_starts(V, n_dw_blocks, s) (multiples of 256,
 *                    the last block ends at V; a block may be empty)
 *   dw_block_events  cudaEvent_t[n_dw_blocks] (entries may be NULL) or NULL
 *   dh_event         cudaEvent_t or NULL
 *   reserve_sms      in [0, SM count - 2]
 * Events belong to the stream's device.  Every event is recorded even when
 * its part is skipped (dH or dW NULL).  Blocking does not change the order in
 * which any dW element is reduced: results are bit-identical to the call
 * without hooks.
 *
 * spo_policy_loss_bwd_ex: spo_policy_loss_bwd (v_offset = 0, dH_fp32 = 0) or
 * spo_policy_loss_bwd_slice (W points at row v_offset of the head; dH_fp32 =
 * 1: dH is fp32, the slice's part), plus hooks (NULL: none).  Workspace as
 * spo_policy_loss_bwd_workspace_size(T, d, V).
 * ------------------------------------------------------------------------- */
typedef struct spo_bwd_hooks {
    int32_t n_dw_blocks;
    int32_t reserve_sms;
    void* const* dw_block_events;
    void* dh_event;
} spo_bwd_hooks;
SPO_API spo_status spo_dw_block_starts(int64_t V, int32_t n_blocks, int64_t* starts);
SPO_API spo_status spo_policy_loss_bwd_ex(const void* H, const void* W, const int32_t* tgt,
                                          const float* lse, const float* g, int64_t T, int64_t d,
                                          int64_t V, int64_t v_offset, float inv_temp, void* dH,
                                          int dH_fp32, float* dW, int accumulate_dW,
                                          const spo_bwd_hooks* hooks, void* ws, size_t ws_bytes,
                                          void* stream);

/* ---------------------------------------------------------------------------
 * Kept-exponential form of a2 + a6: the forward also stores, for every kept
 * token row r and vocabulary entry v, E[r][v] = exp(z - m) in bf16, m the
 * row's largest logit in v's 256-entry vocabulary tile; the backward then forms
 * G = inv_temp * g (onehot - E exp(m - lse)) from E instead of recomputing the
 * logits, and E's buffer becomes G.  This trades T x V x 2 bytes of device
 * memory (5 GB at T = 16384, V = 151936; small beside a GB300's 280 GB) for
 * one of the four T x d x V products.  The default path (spo_logprobs_fwd,
 * spo_policy_loss_bwd) keeps nothing: there the logits never reach memory.
 *
 * spo_logprobs_keep_size: bytes of E for T tokens and V entries (rows padded
 *   to a multiple of 256, V bf16 each).
 * spo_logprobs_fwd_keep: spo_logprobs_fwd plus E (16-byte aligned, >=
 *   spo_logprobs_keep_size bytes); lse must be non-NULL.  E rows follow the
 *   forward's compaction of kept tokens, which stays in `ws`.
 * spo_policy_loss_bwd_kept: the backward of spo_policy_loss_bwd from the kept
 *   forward: `keep` and `fwd_ws` exactly as that forward left them (same T,
 *   d, V; E is overwritten with G), lse from it, g from spo_policy_loss_fwd,
 *   W the same head.  dH bf16[T, d], dW fp32[V, d] (+= if accumulate_dW;
 *   either may be NULL).  Accuracy as spo_policy_loss_bwd (E in bf16 adds one
 *   bf16 rounding to G's).
 * ------------------------------------------------------------------------- */
SPO_API spo_status spo_logprobs_keep_size(int64_t T, int64_t V, size_t* bytes);
SPO_API spo_status spo_logprobs_fwd_keep(const void* H, const void* W, const int32_t* tgt,
                                         const uint8_t* mask, int64_t T, int64_t d, int64_t V,
                                         float inv_temp, float* logp, float* entropy, float* lse,
                                         void* keep, size_t keep_bytes, void* ws, size_t ws_bytes,
                                         void* stream);
SPO_API spo_status spo_policy_loss_bwd_kept(const void* W, const float* lse, const float* g,
                                            int64_t T, int64_t d, int64_t V, float inv_temp,
                                            void* keep, size_t keep_bytes, void* fwd_ws,
                                            size_t fwd_ws_bytes, void* dH, float* dW,
                                            int accumulate_dW, void* stream);

/* ---------------------------------------------------------------------------
 * Vocabulary-split form of a2/a3 and a6-a8: the LM head's V rows split into
 * contiguous slices, one per GPU (tensor-parallel LM head).  The paper trains
 * on two GPUs (section 3, "Base Models") without describing this split; it is
 * the form of the path that shards W instead of the batch.  Because the
 * softmax normaliser couples all V logits of a token, the slices exchange one
 * 16-byte record per token in the forward and sum their dH in the backward:
 *
 *   rank k:  rec_k = spo_logprobs_fwd_slice(H, W[v0_k : v0_k + V_k], ...)
 *   all:     all-gather rec_0 .. rec_{R-1} (T x 16 bytes each)
 *            spo_logprobs_merge_slices -> logp, entropy, lse (identical on every rank)
 *            spo_policy_loss_fwd as in the unsplit path
 *   rank k:  spo_policy_loss_bwd_slice -> dH_k (fp32), dW[v0_k : v0_k + V_k]
 *   all:     all-reduce (sum) of dH_k -> dH; dW stays sharded with W
 *
 * The three calls run on any device; nothing here communicates.
 *
 * spo_logprobs_fwd_slice: the forward over vocabulary rows [v_offset,
 * v_offset + V_slice) of the full head, W_slice pointing at row v_offset.
 * Sizes, alignment, mask and workspace (spo_logprobs_workspace_size(T, d,
 * V_slice)) as in spo_logprobs_fwd with V = V_slice; 0 <= v_offset.  tgt holds
 * ids of the full vocabulary.  Writes rec float32[T][4], 16-byte aligned: for a
 * kept token, with u = z log2(e) over the slice's logits,
 *   rec[t] = { max u,  sum 2^(u - max u),  sum 2^(u - max u) u,
 *              z[tgt[t]] if tgt[t] is in the slice, else -inf }
 * and {0, 0, 0, 0} for a skipped token (mask 0 or tgt < 0).
 * ------------------------------------------------------------------------- */
SPO_API spo_status spo_logprobs_fwd_slice(const void* H, const void* W_slice, const int32_t* tgt,
                                          const uint8_t* mask, int64_t T, int64_t d,
                                          int64_t V_slice, int64_t v_offset, float inv_temp,
                                          float* rec, void* ws, size_t ws_bytes, void* stream);

/* spo_logprobs_merge_slices: rec float32[n_slices][T][4] (the slices' records
 * back to back, in any slice order) -> logp, entropy, lse exactly as
 * spo_logprobs_fwd defines them over the union of the slices.  A token whose
 * records all have a zero second entry (skipped) gets 0.  The slices must
 * together cover the vocabulary once and contain every kept token's target
 * (otherwise that token's logp is -inf).  entropy and lse may be NULL;
 * 1 <= n_slices <= 1024, 1 <= T <= 2^24. */
SPO_API spo_status spo_logprobs_merge_slices(const float* rec, int32_t n_slices, int64_t T,
                                             float* logp, float* entropy, float* lse,
                                             void* stream);

/* spo_policy_loss_bwd_slice: the backward restricted to the slice's columns of
 * G, with lse the full-vocabulary lse from spo_logprobs_merge_slices:
 *   G_k     = inv_temp * g[t] * (1[v0 + j == tgt[t]] - exp(z_t[v0 + j] - lse[t])), j < V_slice
 *   dH_part = G_k W_slice   fp32[T, d] out (the slices' parts sum to dH; NULL to skip)
 *   dW_slice = G_k^T H      fp32[V_slice, d] out (+= if accumulate_dW; NULL to skip)
 * Arguments otherwise as in spo_policy_loss_bwd with V = V_slice; workspace
 * spo_policy_loss_bwd_workspace_size(T, d, V_slice).  Rows with g[t] == 0 get
 * dH_part = 0. */
SPO_API spo_status spo_policy_loss_bwd_slice(const void* H, const void* W_slice,
                                             const int32_t* tgt, const float* lse, const float* g,
                                             int64_t T, int64_t d, int64_t V_slice,
                                             int64_t v_offset, float inv_temp, float* dH_part,
                                             float* dW_slice, int accumulate_dW, void* ws,
                                             size_t ws_bytes, void* stream);

/* ---------------------------------------------------------------------------
 * The whole GRPO step of Eq. 3 in one call: a1 (loss tokens: mask, ignore
 * index, the 1024-token window of section 3) -> a2 + a3 (log-probs over the
 * full vocabulary) -> a4 (group advantages) -> a5 (clipped surrogate, KL,
 * aggregation, g = dL/dlogp) -> a6 - a8 (dH, dW), in stream order, validated
 * once on the host.  Each step computes exactly what the separate calls
 * compute; the backward reuses the forward's compaction of loss tokens
 * instead of compacting again, so loss tokens whose g is exactly 0 (a binding
 * clip with kl_beta = 0) run through the GEMMs with a zero gradient row.
 * With no such token, dH and dW are bit-identical to those of the separate
 * calls on the same inputs.
 *
 * spo_grpo_batch (all DEVICE arrays, as in the separate calls):
 *   H bf16[T, d], W bf16[V, d] (16-byte aligned), tgt int32[T],
 *   mask uint8[T] or NULL (1 = generated token), cu_seqlens int32[n_seq+1],
 *   group_id int32[n_seq] in [0, n_groups), rewards fp32[n_seq] (r_i),
 *   old_logp fp32[T], ref_logp fp32[T] or NULL;
 *   sizes as in spo_logprobs_fwd (T <= 2^24) and spo_policy_loss_fwd.
 * spo_grpo_params: inv_temp (> 0), window (<= 0: no cap), clip_eps in
 *   [0, 1), kl_beta, agg (spo_agg), std_mode (spo_std), adv_eps (>= 0),
 *   loss_scale: DEVICE fp32 scalar multiplying the loss and g (a
 *   data-parallel rank's weight), or NULL for 1.
 * spo_grpo_outputs: loss fp32[1] (required); stats fp32[4] as in
 *   spo_policy_loss_fwd; logp, entropy, lse, g fp32[T], adv fp32[n_seq],
 *   loss_mask uint8[T]; dH bf16[T, d] (16-byte aligned), dW fp32[V, d]
 *   (+= when accumulate_dW).  Every output but loss may be NULL: it is then
 *   kept in the workspace where the step needs it (entropy is then not
 *   computed; dH or dW not at all).
 * hooks: as in spo_policy_loss_bwd_ex, or NULL.
 * ws: >= spo_grpo_workspace_size(T, d, V, n_seq, n_groups) bytes, 256-byte
 *   aligned.
 * ------------------------------------------------------------------------- */
typedef struct spo_grpo_batch {
    const void* H;
    const void* W;
    const int32_t* tgt;
    const uint8_t* mask;
    const int32_t* cu_seqlens;
    const int32_t* group_id;
    const float* rewards;
    const float* old_logp;
    const float* ref_logp;
    int64_t T, d, V;
    int32_t n_seq, n_groups;
} spo_grpo_batch;
typedef struct spo_grpo_params {
    float inv_temp;
    int32_t window;
    float clip_eps;
    float kl_beta;
    int32_t agg;
    int32_t std_mode;
    float adv_eps;
    const float* loss_scale;
} spo_grpo_params;
typedef struct spo_grpo_outputs {
    float* loss;
    float* stats;
    float* logp;
    float* entropy;
    float* lse;
    float* g;
    float* adv;
    uint8_t* loss_mask;
    void* dH;
    float* dW;
    int32_t accumulate_dW;
} spo_grpo_outputs;
SPO_API spo_status spo_grpo_workspace_size(int64_t T, int64_t d, int64_t V, int32_t n_seq,
                                           int32_t n_groups, size_t* bytes);
SPO_API spo_status spo_grpo_step(const spo_grpo_batch* batch, const spo_grpo_params* params,
                                 const spo_grpo_outputs* out, const spo_bwd_hooks* hooks, void* ws,
                                 size_t ws_bytes, void* stream);

/* One workspace for a whole step, under the boundary specification's name:
 * bytes enough for spo_grpo_step with any n_groups <= n_seq, and for any
 * single call of spo_logprobs_fwd, spo_policy_loss_fwd (n_groups <= n_seq),
 * spo_group_advantages_ws and spo_policy_loss_bwd at these sizes, so the
 * separate calls of one step can share it on one stream. */
SPO_API spo_status spo_workspace_size(int64_t T, int64_t d, int64_t V, int32_t n_seq,
                                      size_t* bytes);

/* ---------------------------------------------------------------------------
 * spo_policy_loss_fwd without a caller workspace.  The paper has no
 * counterpart: this is a convenience for callers that cannot hand out device
 * scratch memory -- for example code running under a framework whose memory
 * pool already owns all device memory, or a host that must not call
 * cudaMalloc on this path because it would synchronise the device.  It
 * allocates nothing: its scratch is a 1 MiB array in the library's own device
 * image (present on every GPU that loads libspo, until the process exits).
 *
 * Arguments, results and accuracy are those of spo_policy_loss_fwd minus
 * ws / ws_bytes; inputs and outputs are still the caller's device buffers.
 * Limit: spo_policy_loss_workspace_size(n_seq, n_groups) must be at most
 * 1 MiB (roughly n_seq <= 32000 for a few thousand groups); larger sizes are
 * rejected with SPO_ERR_WORKSPACE before anything is enqueued.
 * The first call on a device looks up the array's device address (with that
 * device current); make that first call before any stream capture.  The
 * scratch used is the current device's copy, so `stream` must belong to the
 * current device: a stream of another device is refused with
 * SPO_ERR_INVALID_ARG.
 * Every call shares the one array, and what is left in it is overwritten or
 * cleared on the stream by the next call: calls that can overlap on the GPU
 * (different streams, or several host threads) race on it and must be
 * serialised by the caller.
 * ------------------------------------------------------------------------- */
SPO_API spo_status spo_policy_loss_fwd_noalloc(const float* logp, const float* old_logp,
                                               const float* ref_logp, const float* adv,
                                               const int32_t* cu_seqlens, const int32_t* group_id,
                                               int32_t n_seq, int32_t n_groups,
                                               const uint8_t* loss_mask, int64_t T, float clip_eps,
                                               float kl_beta, int agg, float* loss, float* g,
                                               float* stats, void* stream);

/* ---------------------------------------------------------------------------
 * Measurement hooks (no counterpart in the paper; used to report per-kernel
 * device time against the tensor-core roofline).
 *
 * spo_trace_enable(1): from now on every launch sequence of this library
 *   (each GEMM, and each small-kernel step) is bracketed by a start/stop CUDA
 *   event pair recorded on the launch stream.  Host-global; two event records
 *   per traced sequence.
 * spo_trace_read: waits for every recorded pair, writes up to max_records
 *   (kind, milliseconds) in launch order, returns the number recorded in
 *   *n_records (may exceed max_records) and clears the record list.  kind:
 *   0 = logits + online logsumexp (a2), 1 = logits recompute -> G (a6),
 *   2 = dH = G W (a7), 3 = dW = G^T H (a8), 4 = split-vocab combine (a3),
 *   5 = forward row selection + gather, 6 = backward row selection + gather,
 *   7 = policy-loss forward (a5), 8 = group advantages (a4),
 *   9 = token selection (a1), 10 = reward composition, 11 = ranker,
 *   12 = merge of vocabulary-slice records, 13 = G formed from a kept forward.
 * spo_launch_count: kernels launched by this library since it was loaded
 *   (host-side counter; every kernel launch adds one).
 * ------------------------------------------------------------------------- */
/* Launch tuning, host-global, for every later call on any device:
 *   SPO_TUNE_PAIR_MMA (default 1): 1 = two CTAs of a cluster share one
 *     256 x 256 tile through a cta_group::2 MMA, 0 = one CTA per 128 x 256 tile.
 *   SPO_TUNE_GROUP_M: tile rows (or columns) walked together by the
 *     persistent raster (L2 reuse of the streamed operand), for every GEMM;
 *     SPO_TUNE_GROUP_M_FWD / _GRAD / _DH / _DW set one GEMM (trace kinds 0-3;
 *     defaults 16, 16, 8, 8).
 *   SPO_TUNE_RASTER: 0 = groups of tile rows, 1 = groups of tile columns, for
 *     every GEMM; SPO_TUNE_RASTER_FWD / _GRAD / _DH / _DW one GEMM (defaults
 *     0, 0, 0, 1).
 *   SPO_TUNE_DYNAMIC_MASK (default 15): bit k set = GEMM kind k (trace kinds
 *     0-3) takes its tiles in raster order from an atomic counter instead of
 *     a static round robin, so in-flight tiles stay a contiguous window.
 *   SPO_TUNE_DW_SPLIT_ROWS (default 8192; multiple of 256, 0 = off): dW =
 *     G^T H is reduced over at most this many token rows per pass, later
 *     passes adding into dW (smaller operand slabs stay in L2).
 *   SPO_TUNE_KSYNC_FWD / _GRAD / _DH / _DW (default 0 = off): a k-progress
 *     throttle for one GEMM kind: each CTA pair publishes the k-blocks (64
 *     elements of the reduction) it has issued and does not run more than
 *     this many ahead of the slowest pair, so the pairs whose tiles share an
 *     operand slab read it close together in time (from L2).  The waits are
 *     bounded (20 us); results do not depend on the setting.
 *   SPO_TUNE_KSYNC_EPOCH (default 16): k-blocks between two throttle checks.
 *   SPO_TUNE_DH_WIDE (default 1): dH with 256 x 512 output tiles per CTA
 *     pair (two N = 256 MMAs per k-step into both TMEM accumulators; the
 *     tiles of the last round split into 256-column halves), pair mode only:
 *     0 = never (256 x 256), 1 = when V >= 32768 (long reductions, where the
 *     epilogue no longer overlapping the next tile's MMAs costs nothing),
 *     2 = always.  A wave reads G's row slabs half as often.  Results are
 *     bit-identical either way.
 *   SPO_TUNE_LOGITS_WIDE (default 6): the logits GEMMs with 256 x 512 tiles,
 *     bit 0 the forward (logits + logsumexp) in every call, bit 1 the
 *     backward's recompute (G), bit 2 the forward inside spo_grpo_step (where
 *     it shares the power budget with the backward; alone, at full clock, the
 *     256 x 256 tile is faster); pair mode only.  The two accumulator halves
 *     are drained one after the other while MMAs fill the other half.
 *     Results are bit-identical either way.
 *   SPO_TUNE_DEFAULTS (value ignored): every setting back to its default.
 * Results do not depend on any setting beyond fp32 summation order. */
typedef enum spo_tune_key {
    SPO_TUNE_PAIR_MMA = 0,
    SPO_TUNE_GROUP_M = 1,
    SPO_TUNE_RASTER = 2,
    SPO_TUNE_DYNAMIC_MASK = 3,
    SPO_TUNE_DW_SPLIT_ROWS = 4,
    SPO_TUNE_GROUP_M_FWD = 5,
    SPO_TUNE_GROUP_M_GRAD = 6,
    SPO_TUNE_GROUP_M_DH = 7,
    SPO_TUNE_GROUP_M_DW = 8,
    SPO_TUNE_RASTER_FWD = 9,
    SPO_TUNE_RASTER_GRAD = 10,
    SPO_TUNE_RASTER_DH = 11,
    SPO_TUNE_RASTER_DW = 12,
    SPO_TUNE_DEFAULTS = 13,
    SPO_TUNE_KSYNC_FWD = 14,
    SPO_TUNE_KSYNC_GRAD = 15,
    SPO_TUNE_KSYNC_DH = 16,
    SPO_TUNE_KSYNC_DW = 17,
    SPO_TUNE_KSYNC_EPOCH = 18,
    SPO_TUNE_DH_WIDE = 19,
    SPO_TUNE_LOGITS_WIDE = 20
} spo_tune_key;
SPO_API spo_status spo_set_tuning(int key, int64_t value);

SPO_API spo_status spo_trace_enable(int on);
SPO_API spo_status spo_trace_read(int* kinds, float* ms, int max_records, int* n_records);
SPO_API long long spo_launch_count(void);

#ifdef __cplusplus
}
#endif

#endif /* SPO_H_ */
