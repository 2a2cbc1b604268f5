// gemm.h -- the tensor-core GEMM kernel's interface: tile geometry, the
// epilogue kinds, the launch arguments, tensor-map encoding and the launcher.
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

// Default launch schedule per GEMM kind (0 logits + logsumexp, 1 recompute
// -> G, 2 dH, 3 dW), from DRAM-traffic sweeps: the logits GEMMs walk 16 tile
// rows together, dH (whose 256 x 512 tiles reduce over the whole vocabulary)
// 8, dW groups of 8 tile columns; every GEMM takes its tiles from an atomic
// counter; dW reduces over passes of at most 8192 token rows.
constexpr int kDefaultGroupM[4] = {16, 16, 8, 8};
constexpr int kDefaultRaster[4] = {0, 0, 0, 1};
constexpr int kDefaultDynamicMask = 0xF;
constexpr int kDefaultDwSplitRows = 8192;
// Ints of workspace reserved for the k-progress throttle's state (two u64), its
// default window per GEMM kind in k-blocks (0 = off) and its check interval.
constexpr int kKsyncSlots = 4;
constexpr int kDefaultKsync[4] = {0, 0, 0, 0};
constexpr int kDefaultKsyncEpoch = 16;
// dH with 256 x 512 tiles per CTA pair: 0 never, 1 when the reduction (the
// vocabulary rows) is at least kDhWideMinK, 2 always.  A wide tile holds both
// TMEM accumulators, so its epilogue no longer overlaps the next tile's MMAs:
// negligible at K = 151936 (1.5 ms of MMA per tile), a few % at K = 8192.
constexpr int kDefaultDhWide = 1;
constexpr int kDhWideMinK = 32768;
// The logits GEMMs with 256 x 512 tiles: bit 0 the forward in every call, bit
// 1 the recompute, bit 2 the forward inside spo_grpo_step.  At K = d = 5120 a
// wide tile's epilogue overlaps the MMAs only through the split drain of its
// two halves.  The forward's epilogue outlasts that (a few % slower alone at
// full clock, where a forward-only call runs), the recompute's does not; in
// the power-capped step both wide tiles leave more of the budget to the
// kernels around them.
constexpr int kDefaultLogitsWide = 6;

// What the epilogue does with a finished 128 x 256 fp32 accumulator tile.
enum EpiKind : int {
  EPI_LSE = 0,   // online max / sum-exp / sum-exp*z per row + target logit -> partials
  EPI_GRAD = 1,  // G = scale * g_row * (onehot - exp(scale*acc - lse_row)) -> bf16
  EPI_DH = 2,    // bf16 rows scattered to row_idx[row]
  EPI_DW = 3,    // fp32 rows, overwrite or accumulate
  EPI_LSE_KEEP = 4,  // EPI_LSE, and E = 2^(t - tile max) kept in bf16 for the backward
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
  // k-progress throttle (NULL = off): 16 zeroed, 8-byte aligned bytes holding
  // the running units' summed k-block progress and their count; a unit stays
  // at most ksync_window k-blocks ahead of the average (bounded wait), checked
  // every ksync_epoch k-blocks.  Affects timing and L2 reuse only.
  int* kprog;
  int ksync_window;
  int ksync_epoch;
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
  // NULL: lse and gvec are indexed by row; else by vec_idx[row] (token
  // positions of the compacted rows, so the vectors need no gather)
  const int* vec_idx;
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

// Supported (epi, a_mn, b_mn): (LSE,0,0) (LSE_KEEP,0,0) (GRAD,0,0) (DH,0,1)
// (DW,1,1).  With `pair` the grid must be even (clusters of two CTAs).  tc is
// the output's tensor map for the TMA-store epilogues (GRAD and LSE_KEEP: G or
// E as bf16, box 64 x 32; DW: dW as fp32, box 32 x 32; all 128-byte swizzled);
// ignored by LSE and DH.
constexpr uint32_t kStoreBoxRows = 32;
// One thread waits on a barrier nothing arrives on (bounded-wait self-test).
cudaError_t launch_bounded_wait_selftest(int* err, cudaStream_t s);

// wide: dH (EPI_DH, MN-major B) in pair mode with 256 x 512 tiles (the last
// round's tiles split in 256-column halves); ignored for every other case.
cudaError_t launch_gemm(int epi, bool a_mn, bool b_mn, bool pair, const CUtensorMap& ta,
                        const CUtensorMap& tb, const CUtensorMap& tc, const GemmArgs& args, int grid,
                        cudaStream_t s, bool wide = false);

}  // namespace spo
