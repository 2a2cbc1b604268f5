// internal.h -- interface between the C-ABI layer (api.cu) and the kernels.
// Not part of the public ABI.
#pragma once

#include "gemm.h"

namespace spo {

// SM count of the current device, cached per ordinal (1 if the query fails).
int sm_count();

// ---------------------------------------------------------------- small kernels
// Compaction of selected rows: kind 0 selects (mask == NULL || mask[t]) &&
// tgt[t] >= 0, kind 1 selects g[t] != 0.  Writes idx[0..count) ascending and
// *count.  scratch holds 2 * compact_blocks(T) ints.
int compact_blocks(long long T);
cudaError_t launch_compact(int kind, const uint8_t* mask, const int* tgt, const float* g,
                           long long T, int* scratch, int* idx, int* count, cudaStream_t s);

// Hc[r] = H[idx[r]] for r < count and 0 for count <= r < round_up(count, kRowPad)
// (r < rows_cap); also gathers up to three per-row vectors (NULL to skip).
// tgt_c[r] = tgt[idx[r]] - tgt_off when that lies in [0, tgt_lim), else -1 (the
// target is outside this vocabulary slice: no logit of the slice is the target).
cudaError_t launch_gather(const __nv_bfloat16* H, int d, const int* idx, const int* count,
                          int rows_cap, __nv_bfloat16* Hc, const int* tgt, int* tgt_c,
                          long long tgt_off, long long tgt_lim, const float* a, float* a_c,
                          const float* b, float* b_c, cudaStream_t s);

// Merges each kept row's vocab-tile partials.  With rec == NULL writes logp,
// entropy, lse at the row's token position; otherwise writes the slice record
// rec[t] = (m, s, e, z_tgt) (log2 units for m and e; z_tgt natural, -inf when
// tgt_c < 0) and leaves the three outputs untouched.
cudaError_t launch_lse_combine(const float* partials, int nsplit,
                               const float* ztgt, const int* idx, const int* count,
                               int rows_cap, float* logp, float* entropy, float* lse,
                               const int* tgt_c, float4* rec, cudaStream_t s);

// G from the kept forward, in place in E (bf16 [rows][ldE], V % 8 == 0):
// rows r < *count of the forward's compaction (idx, compacted targets tgt_c),
// lse and g at token positions, partials the forward's (first plane: the
// per-tile max in log2 units).
cudaError_t launch_form_g(__nv_bfloat16* E, long long ldE, int V, int rows_cap,
                          const float* partials, int nsplit, const int* idx, const int* count,
                          const int* tgt_c, const float* lse, const float* g, float inv_temp,
                          cudaStream_t s);

// Merges n_slices slice records per token, rec[k * T + t], into logp, entropy
// and lse; a token whose records all have s == 0 (skipped) gets 0.
cudaError_t launch_merge_slices(const float4* rec, int n_slices, long long T, float* logp,
                                float* entropy, float* lse, cudaStream_t s);

cudaError_t launch_token_select(const int* cu_seqlens, const uint8_t* mask, const int* tgt,
                                int n_seq, int window, uint8_t* loss_mask, int* n_tok,
                                cudaStream_t s);

cudaError_t launch_group_advantages(const float* rewards, const int* group_id, int n_seq,
                                    int n_groups, int std_mode, float eps, float* adv,
                                    cudaStream_t s);
// The same advantages in O(n_seq + n_groups) when every group's members are
// contiguous (one run of equal ids), falling back to the per-group scan
// otherwise; ws holds adv_ws_bytes(n_groups) bytes.
size_t adv_ws_bytes(int n_groups);
cudaError_t launch_group_advantages_runs(const float* rewards, const int* group_id, int n_seq,
                                         int n_groups, int std_mode, float eps, float* adv,
                                         void* ws, cudaStream_t s);

// Composite reward (section 2.2 verifiable reward + structural score).
struct RewardParams {
  float alpha_comp, alpha_wrong, alpha_speed, alpha_cv, s_min, s_max;
};
cudaError_t launch_reward_compose(const uint8_t* compiled, const float* pass_rate,
                                  const float* speedup, const float* cv, const float* r_struct,
                                  int n, const RewardParams& q, float* out, cudaStream_t s);

// Offline structural ranker: 11 -> 64 -> 32 -> 1 ReLU MLP, packed parameters
// W1[64][11], b1[64], W2[32][64], b2[32], w3[32], b3.
constexpr int kRankerFeatures = 11;
constexpr int kRankerParams = 64 * 11 + 64 + 32 * 64 + 32 + 32 + 1;  // 2881
int ranker_blocks(int n_pairs);
size_t ranker_ws_bytes(int n_pairs);
cudaError_t launch_ranker_scores(const float* phi, const float* mu, const float* sigma, int n,
                                 const float* params, float* scores, cudaStream_t s);
cudaError_t launch_ranker_pair_loss(const float* phi, const float* mu, const float* sigma,
                                    const int* pos, const int* neg, int n_pairs,
                                    const float* params, const uint8_t* keep1,
                                    const uint8_t* keep2, float drop_p, float* loss, float* grad,
                                    float* ws, cudaStream_t s);

// x[i] *= alpha (alpha read from device memory when alpha_dev != NULL).
// launch_scale_ratio: x[i] *= num[0] / den[0] (fp64 device scalars; 0 when den is 0).
cudaError_t launch_scale_ratio(float* x, long long n, const double* num, const double* den,
                               cudaStream_t s);
cudaError_t launch_scale(float* x, long long n, float alpha, const float* alpha_dev, cudaStream_t s);

// Zeroes row t of out (row_bytes per row, a multiple of 16; out 16-byte aligned)
// for every t < T with g[t] == 0: the dH rows the backward's compaction skips.
cudaError_t launch_zero_skipped_rows(const float* g, long long T, int row_bytes, void* out,
                                     cudaStream_t s);

// Counts of invalid device inputs into counts[6] (zeroed here first); see spo_validate_inputs.
cudaError_t launch_validate(const int* tgt, long long T, long long V, const int* cu, int n_seq,
                            const int* gid, int n_groups, const float* rewards, const float* old_logp,
                            const float* ref_logp, const uint8_t* mask, int* counts, cudaStream_t s);

struct LossWs {
  unsigned long long* scal;  // [4]: non-empty groups, total loss tokens (token mean), ticket,
                             // grid-barrier arrivals
  int* gsize;                // [n_groups]
  int* n_tok;                // [n_seq]
  float2* part_l;            // [n_seq]: c_i * sum of the sequence's l_t as a (hi, lo) pair
  float2* part_rk;           // [n_seq]: sums of rho and of kl
  int* part_clip;            // [n_seq]
  void* bpart;               // [<= 1024]: first-stage sums of the final reduction
};
size_t loss_ws_bytes(int n_seq, int n_groups);
LossWs carve_loss_ws(void* ws, int n_seq, int n_groups);

// The loss forward (group counts, token pass, fixed-order sum) as one
// cooperative launch; err is the device error word (a grid barrier that
// expires records its code there).  cscale (device scalar or NULL)
// multiplies every c_t.  With `rewards` non-NULL the launch first computes the
// group advantages into adv_out (the per-group scan of
// launch_group_advantages, the same bits) and uses them; `adv` is then unused.
cudaError_t launch_policy_loss(const float* logp, const float* old_logp, const float* ref_logp,
                               const float* adv, const int* cu_seqlens, const int* group_id,
                               int n_seq, int n_groups, const uint8_t* loss_mask, long long T,
                               float clip_eps, float kl_beta, int agg, float* loss, float* g,
                               float* stats, const LossWs& w, cudaStream_t s, int* err,
                               const float* cscale = nullptr, const float* rewards = nullptr,
                               int std_mode = 0, float adv_eps = 0.f, float* adv_out = nullptr);

}  // namespace spo
