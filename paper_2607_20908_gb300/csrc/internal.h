// internal.h -- interface between the C-ABI layer (api.cu) and the kernels.
// Not part of the public ABI.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace spo {

// Tensor-core tile: 128 accumulator rows x 256 columns per CTA, K staged 64
// at a time (one 128-byte swizzle atom of bf16).  In pair mode two CTAs share
// one 256 x 256 tile.
constexpr int BM = 128;
constexpr int BN = 256;
constexpr int BK = 64;
// Compacted row buffers are padded (and zero-filled) to this many rows so a
// pair tile never reads rows past the buffer.
constexpr int kRowPad = 256;
// Floats of logsumexp partials per 32 rows and vocab tile: three planes of 32.
constexpr int kPartialBlock = 96;

// What the epilogue does with a finished 128 x 256 fp32 accumulator tile.
enum EpiKind : int {
  EPI_LSE = 0,   // online max / sum-exp / sum-exp*z per row + target logit -> partials
  EPI_GRAD = 1,  // G = scale * g_row * (onehot - exp(scale*acc - lse_row)) -> bf16
  EPI_DH = 2,    // bf16 rows scattered to row_idx[row]
  EPI_DW = 3,    // fp32 rows, overwrite or accumulate
};

struct GemmArgs {
  // rows M: m_static, or clamp(*m_count - m_offset, 0, m_cap) read on the device
  int m_static;
  const int* m_count;
  int m_offset;
  int m_cap;
  int n;  // columns N
  // reduction length K: k_static, or clamp(*k_count - k_offset, 0, k_cap) on the device
  int k_static;
  const int* k_count;
  int k_offset;
  int k_cap;
  int group_m;  // tile rows (raster 0) or columns (raster 1) walked together
  int raster;   // 0: groups of tile rows, 1: groups of tile columns
  int* tile_counter;  // zeroed int: tiles are taken in raster order from it; NULL = static
  float scale;  // inv_temp for EPI_LSE / EPI_GRAD
  // EPI_LSE
  const int* tgt;     // target id of each row
  // Per (row, vocab tile) partials m = max*log2e, s = sum 2^(t-m), e = sum 2^(t-m) t, laid out
  // [row / 32][vocab tile][m, s, e][row % 32] (kPartialBlock floats per 32 rows and tile).
  float* partials;
  int nsplit;  // number of vocab tiles, ceil(n / BN)
  float* ztgt;        // target logit (natural units) of each row
  // EPI_GRAD
  const float* lse;   // natural-log lse of each row
  const float* gvec;  // dL/dlogp of each row
  __nv_bfloat16* G;   // [rows][ldG]
  long long ldG;
  // EPI_DH: rows scattered to row_idx[row], bf16 to out_bf16 or, when out_f32
  // is set, fp32 to out_f32 (the per-slice partial of the vocabulary split)
  const int* row_idx;         // output row of each row (NULL: identity)
  __nv_bfloat16* out_bf16;
  long long ld_out;
  // EPI_DW (the output itself goes through the tc tensor map)
  float* out_f32;
  int accumulate;  // 1: reduce-add into the output, 0: overwrite
  int* err;  // device error word
};

size_t gemm_smem_bytes(bool pair);
int gemm_tile_m(bool pair);        // output rows per tile (128 solo, 256 pair)
int gemm_b_box_rows(bool pair);    // rows of a K-major B operand staged per CTA

// Host-side count of kernels this library has launched (for launch accounting).
void note_launches(int n);
long long launches();

// Encodes a 2-D bf16 tensor map with 128-byte swizzle.  inner/outer are the
// extents in elements / rows, row_bytes the pitch, box the staged tile.
cudaError_t make_tmap_bf16(CUtensorMap* tm, const void* base, uint64_t inner, uint64_t outer,
                           uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer);
cudaError_t make_tmap_f32(CUtensorMap* tm, const void* base, uint64_t inner, uint64_t outer,
                          uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer);

// Supported (epi, a_mn, b_mn): (LSE,0,0) (GRAD,0,0) (DH,0,1) (DW,1,1).  With
// `pair` the grid must be even (clusters of two CTAs).  tc is the output's
// tensor map for the TMA-store epilogues (GRAD: G as bf16, box 64 x 32; DW:
// dW as fp32, box 32 x 32; both 128-byte swizzled); ignored by LSE and DH.
constexpr uint32_t kStoreBoxRows = 32;
cudaError_t launch_gemm(int epi, bool a_mn, bool b_mn, bool pair, const CUtensorMap& ta,
                        const CUtensorMap& tb, const CUtensorMap& tc, const GemmArgs& args, int grid,
                        cudaStream_t s);

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
cudaError_t launch_scale(float* x, long long n, float alpha, const float* alpha_dev, cudaStream_t s);

// Counts of invalid device inputs into counts[6] (zeroed here first); see spo_validate_inputs.
cudaError_t launch_validate(const int* tgt, long long T, long long V, const int* cu, int n_seq,
                            const int* gid, int n_groups, const float* rewards, const float* old_logp,
                            const float* ref_logp, const uint8_t* mask, int* counts, cudaStream_t s);

struct LossWs {
  int* gsize;                // [n_groups]
  int* n_tok;                // [n_seq]
  unsigned long long* scal;  // [2]: non-empty groups, total loss tokens
  double* part;              // [n_seq][3]: sum c*l, sum rho, sum kl
  int* part_clip;            // [n_seq]
  double* bpart;             // [64][4]: first-stage sums of the final reduction
};
size_t loss_ws_bytes(int n_seq, int n_groups);
LossWs carve_loss_ws(void* ws, int n_seq, int n_groups);

cudaError_t launch_policy_loss(const float* logp, const float* old_logp, const float* ref_logp,
                               const float* adv, const int* cu_seqlens, const int* group_id,
                               int n_seq, int n_groups, const uint8_t* loss_mask, long long T,
                               float clip_eps, float kl_beta, int agg, float* loss, float* g,
                               float* stats, const LossWs& w, cudaStream_t s);

}  // namespace spo
