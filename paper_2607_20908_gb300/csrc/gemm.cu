// gemm.cu -- persistent, warp-specialised tcgen05 GEMM for sm_103a with the
// fused epilogues of the GRPO log-prob path.
//
//   C[M, N] = A[M, K] * B[N, K]^T    (bf16 in, fp32 accumulate in TMEM)
//
// One CTA per SM.  By default two CTAs of a cluster share each 256 x 256
// output tile through a cta_group::2 MMA (each stages 128 rows of A and half
// of the tile's B rows); with SPO_TUNE_PAIR_MMA = 0 a CTA owns a 128 x 256
// tile alone.  Warp 0 issues TMA loads into a shared-memory ring (7 stages of
// 32 KB per CTA in pair mode, 6 when the epilogue stages its TMA stores, 4 of
// 48 KB alone), warp 1 issues tcgen05.mma from one thread into one of two TMEM
// accumulators (2 x 256 columns), and warps 2-5 drain the other accumulator
// through the epilogue, so MMA and epilogue overlap.  Wide tiles (dH and the
// recompute, pair mode) are 256 x 512: two N = 256 MMAs per k-step fill both
// accumulators from a ring of 4 stages of 48 KB, and the two halves are
// drained one after the other while MMAs fill the other half.  Tiles are taken in a
// grouped raster order, statically or from an atomic counter whose values the
// leader's producer publishes to both CTAs through a shared-memory ring.
// Operands may be K-major (rows of K contiguous) or MN-major (rows of M or N
// contiguous); both are staged with the 128-byte swizzle.
//
// The epilogues are the four places where the path touches the logits:
//   EPI_LSE  : forward. Online max / sum-exp / sum-exp*z of each row over the
//              tile plus the target logit; writes one partial per
//              (vocab tile, row).  The logits themselves never leave TMEM.
//   EPI_GRAD : backward. G = inv_temp * g_t * (onehot - exp(z - lse_t)) in
//              bf16, through TMA bulk stores.
//   EPI_DH   : dH = G W rows scattered back to token rows, bf16 (or fp32 for
//              one vocabulary slice's part).
//   EPI_DW   : dW = G^T H, fp32 through TMA bulk stores or reduce-adds.
#include <math.h>

#include "gemm.h"
#include "tc.cuh"

namespace spo {

namespace {

constexpr uint32_t MN_BLOCK_BYTES = 64 * BK * 2;   // [BK rows][64 MN] block, 8 KB
constexpr int NUM_THREADS = 192;
constexpr float kLog2e = 1.4426950408889634f;

__device__ __forceinline__ int clampi(int v, int lo, int hi) { return v < lo ? lo : (v > hi ? hi : v); }

// Grouped raster.  raster 0: `gm` tile rows are walked together across all
// tile columns, so the A rows of a group stay in L2 while B streams past them.
// raster 1: the same with the roles of rows and columns exchanged.
__device__ __forceinline__ void tile_coords(int tile, int mt, int nt, int gm, int raster, int& mb,
                                            int& nb) {
  const int outer = raster ? nt : mt;
  const int inner = raster ? mt : nt;
  const int per_group = gm * inner;
  const int group = tile / per_group;
  const int first = group * gm;
  const int size = min(gm, outer - first);
  const int in = tile - group * per_group;
  const int o = first + in % size;
  const int i = in / size;
  mb = raster ? i : o;
  nb = raster ? o : i;
}

// The k-progress throttle.  kstate[0] holds the k-blocks issued so far by the
// units (CTA pairs, or CTAs) that are running, kstate[1] how many are running.
// A unit adds its progress every `epoch` k-blocks and waits (bounded) while
// it is more than `window` k-blocks ahead of the running units' average, so
// the units whose tiles share operand slabs read them close together in time,
// from L2 instead of DRAM.  One fire-and-forget add and two loads per check.
// A wait gives up after kKsyncMaxWaitNs (a unit not yet resident, another
// kernel on the SMs): results never depend on the throttle.
constexpr unsigned long long kKsyncMaxWaitNs = 20000ull;  // 20 us

// Wide tiles: k-blocks at each end of a tile whose two accumulator halves are
// issued one after the other, so each half's drain overlaps MMAs (fewer than
// the four stages of a wide ring, which hold them meanwhile).
constexpr int kWideOverlap = 3;

__device__ __forceinline__ void ksync_wait(unsigned long long* kstate, long long prog, int window) {
  const unsigned long long t0 = globaltimer();
  for (;;) {
    const long long sum = static_cast<long long>(ld_relaxed_gpu_u64(kstate));
    const long long active = static_cast<long long>(ld_relaxed_gpu_u64(kstate + 1));
    if (active <= 0 || prog * active <= sum + static_cast<long long>(window) * active) return;
    if (globaltimer() - t0 > kKsyncMaxWaitNs) return;
    __nanosleep(128);
  }
}

// 2^x by the SFU's own instruction (PTX ex2.approx.ftz.f32: relative error
// about 2^-22, subnormal results flushed to zero, 2^-inf = 0), without the
// range handling of the exp2f library call around it.  The logits epilogues
// take one per logit; without that handling their ALU work drops by a sixth.
__device__ __forceinline__ float ex2_sfu(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&h);
}

// ------------------------------------------------------------ epilogues
// Each thread owns one accumulator row (TMEM lane) and walks its 256 columns
// in 8 chunks of 32.

__device__ __forceinline__ void epi_lse(const GemmArgs& p, uint32_t taddr, int row, int M, int nb) {
  const bool row_ok = row < M;
  const int y = row_ok ? p.tgt[row] : -1;
  const float sc2 = p.scale * kLog2e;  // logits in log2 units: t = z * log2(e)
  const int col_base = nb * BN;
  const bool full = col_base + BN <= p.n;
  float run_m = -INFINITY, run_s = 0.f, run_e = 0.f, zt = 0.f;
  bool hit = false;
#pragma unroll 1
  for (int c = 0; c < BN / 32; ++c) {
    float v[32];
    tmem_ld32(taddr + c * 32, v);
    const int c0 = col_base + c * 32;
    if (y >= c0 && y < c0 + 32) {
#pragma unroll
      for (int j = 0; j < 32; ++j)
        if (c0 + j == y) zt = v[j] * p.scale;
      hit = true;
    }
    float cm = -INFINITY;
    if (full) {
#pragma unroll
      for (int j = 0; j < 32; ++j) cm = fmaxf(cm, v[j]);
    } else {
#pragma unroll
      for (int j = 0; j < 32; ++j)
        if (c0 + j < p.n) cm = fmaxf(cm, v[j]);
    }
    if (c0 >= p.n) continue;  // chunk entirely past the vocabulary (warp-uniform)
    const float nm = fmaxf(run_m, cm * sc2);
    const float r = ex2_sfu(run_m - nm);
    run_s *= r;
    run_e *= r;
    if (full) {
#pragma unroll
      for (int j = 0; j < 32; ++j) {
        const float t = v[j] * sc2;
        const float e = ex2_sfu(t - nm);
        run_s += e;
        run_e = fmaf(e, t, run_e);
      }
    } else {
#pragma unroll
      for (int j = 0; j < 32; ++j) {
        if (c0 + j < p.n) {
          const float t = v[j] * sc2;
          const float e = ex2_sfu(t - nm);
          run_s += e;
          run_e = fmaf(e, t, run_e);
        }
      }
    }
    run_m = nm;
  }
  if (row_ok) {
    float* q = p.partials + (static_cast<size_t>(row >> 5) * p.nsplit + nb) * kPartialBlock +
               (row & 31);
    q[0] = run_m;    // each of the three stores is one 128-byte line per warp
    q[32] = run_s;
    q[64] = run_e;
    if (hit) p.ztgt[row] = zt;
  }
}

// Columns [col_base, col_base + ncols) of the tile, TMEM columns from taddr.
__device__ __forceinline__ void epi_dh(const GemmArgs& p, uint32_t taddr, int row, int M, int col_base,
                                       int ncols) {
  const bool row_ok = row < M;
  const int out_row = row_ok ? (p.row_idx ? p.row_idx[row] : row) : 0;
  const size_t off = static_cast<size_t>(out_row) * p.ld_out;
  __nv_bfloat16* dst = p.out_f32 ? nullptr : p.out_bf16 + off;
  float* dst32 = p.out_f32 ? p.out_f32 + off : nullptr;
#pragma unroll 1
  for (int c = 0; c < ncols / 32; ++c) {
    const int c0 = col_base + c * 32;
    if (c0 >= p.n) break;
    float v[32];
    tmem_ld32(taddr + c * 32, v);
    if (!row_ok) continue;
    if (p.out_f32) {
#pragma unroll
      for (int q = 0; q < 8; ++q)
        if (c0 + 4 * q < p.n)
          *reinterpret_cast<float4*>(dst32 + c0 + 4 * q) =
              make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
      continue;
    }
    uint32_t pk[16];
#pragma unroll
    for (int j = 0; j < 16; ++j) pk[j] = pack_bf16x2(v[2 * j], v[2 * j + 1]);
#pragma unroll
    for (int q = 0; q < 4; ++q)
      if (c0 + 8 * q < p.n)
        *reinterpret_cast<uint4*>(dst + c0 + 8 * q) =
            make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
  }
}

// TMA-store epilogues: each epilogue warp stages its 32 rows x 128 bytes in a
// [32][128 B] shared slot with the 128-byte swizzle (chunk j of row r at
// position j ^ (r % 8): conflict-free writes, and the layout a swizzled
// tensor map expects), then one lane issues a bulk tensor store (or
// reduce-add) of the 32 x 128 B box.  Two slots per warp alternate.
constexpr uint32_t kEpiSlotBytes = 32 * 128;

__device__ __forceinline__ void stage_row128(uint8_t* slot, int lane, const uint32_t (&w)[32]) {
  uint4* row = reinterpret_cast<uint4*>(slot + lane * 128);
#pragma unroll
  for (int j = 0; j < 8; ++j)
    row[j ^ (lane & 7)] = make_uint4(w[4 * j], w[4 * j + 1], w[4 * j + 2], w[4 * j + 3]);
}

// Hands slot (slab & 1) back after staging: fence the generic writes for the
// async proxy, then one lane issues the store.  `reduce` selects add.
__device__ __forceinline__ void flush_slot(const CUtensorMap* tm, uint8_t* slot, int x, int y,
                                           bool reduce, int lane) {
  fence_proxy_async_smem();
  __syncwarp();
  if (lane == 0) {
    if (reduce)
      tma_reduce_add_2d(tm, slot, x, y);
    else
      tma_store_2d(tm, slot, x, y);
    bulk_commit();
  }
}

__device__ __forceinline__ uint8_t* acquire_slot(uint8_t* slots, int slab, int lane) {
  if (lane == 0) bulk_wait_read<1>();  // the store issued from this slot two slabs ago has read it
  __syncwarp();
  return slots + (slab & 1) * kEpiSlotBytes;
}

// G rows as bf16 through 64-column (128-byte) slabs.
__device__ __forceinline__ void epi_grad_tma(const GemmArgs& p, const CUtensorMap* tmC, uint32_t taddr,
                                             int row, int row0, int M, int nb, uint8_t* slots,
                                             int& slab, int lane) {
  const bool row_ok = row < M;
  const int vrow = row_ok && p.vec_idx ? p.vec_idx[row] : row;
  const float gl = row_ok ? p.gvec[vrow] : 0.f;
  const float l2 = row_ok ? p.lse[vrow] * kLog2e : 0.f;
  const int y = row_ok ? p.tgt[row] : -1;
  const float coef = p.scale * gl;
  const float sc2 = p.scale * kLog2e;
  const int col_base = nb * BN;
#pragma unroll 1
  for (int c2 = 0; c2 < BN / 64; ++c2) {
    const int c0 = col_base + c2 * 64;
    if (c0 >= p.n) break;  // warp-uniform; columns past n inside a slab are clipped by the store
    uint32_t w[32];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      float v[32];
      tmem_ld32(taddr + c2 * 64 + h * 32, v);
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const int ca = c0 + h * 32 + 2 * j;
        const float pa = ex2_sfu(fmaf(v[2 * j], sc2, -l2));
        const float pb = ex2_sfu(fmaf(v[2 * j + 1], sc2, -l2));
        w[h * 16 + j] = pack_bf16x2(coef * ((ca == y ? 1.f : 0.f) - pa),
                                    coef * ((ca + 1 == y ? 1.f : 0.f) - pb));
      }
    }
    uint8_t* slot = acquire_slot(slots, slab, lane);
    stage_row128(slot, lane, w);
    flush_slot(tmC, slot, c0, row0, false, lane);
    ++slab;
  }
}

// dW rows as fp32 through 32-column (128-byte) slabs; accumulate = reduce-add.
__device__ __forceinline__ void epi_dw_tma(const GemmArgs& p, const CUtensorMap* tmC, uint32_t taddr,
                                           int row0, int nb, bool kzero, uint8_t* slots, int& slab,
                                           int lane) {
  const int col_base = nb * BN;
#pragma unroll 1
  for (int c = 0; c < BN / 32; ++c) {
    const int c0 = col_base + c * 32;
    if (c0 >= p.n) break;
    float v[32];
    if (kzero) {
#pragma unroll
      for (int j = 0; j < 32; ++j) v[j] = 0.f;
    } else {
      tmem_ld32(taddr + c * 32, v);
    }
    uint32_t w[32];
#pragma unroll
    for (int j = 0; j < 32; ++j) w[j] = __float_as_uint(v[j]);
    uint8_t* slot = acquire_slot(slots, slab, lane);
    stage_row128(slot, lane, w);
    flush_slot(tmC, slot, c0, row0, p.accumulate != 0, lane);
    ++slab;
  }
}

// Forward that also keeps E[row][v] = 2^(t_v - m) in bf16 for the backward
// (t = scale * z * log2 e, m the row's max over this vocabulary tile): one pass
// over the accumulator for m, a second for the sums of epi_lse (now taken
// against the final m) and for E, staged 64 columns at a time for the TMA
// store.  Columns past n are staged as 0 and clipped by the store.
__device__ __forceinline__ void epi_lse_keep(const GemmArgs& p, const CUtensorMap* tmC,
                                             uint32_t taddr, int row, int row0, int M, int nb,
                                             uint8_t* slots, int& slab, int lane) {
  const bool row_ok = row < M;
  const int y = row_ok ? p.tgt[row] : -1;
  const float sc2 = p.scale * kLog2e;
  const int col_base = nb * BN;
  float mx = -INFINITY;
#pragma unroll 1
  for (int c = 0; c < BN / 32; ++c) {
    const int c0 = col_base + c * 32;
    if (c0 >= p.n) break;  // warp-uniform
    float v[32];
    tmem_ld32(taddr + c * 32, v);
#pragma unroll
    for (int j = 0; j < 32; ++j)
      if (c0 + j < p.n) mx = fmaxf(mx, v[j]);
  }
  const float m2 = mx * sc2;  // scale > 0: the max of the scaled logits
  float run_s = 0.f, run_e = 0.f, zt = 0.f;
  bool hit = false;
#pragma unroll 1
  for (int c2 = 0; c2 < BN / 64; ++c2) {
    const int c0 = col_base + c2 * 64;
    if (c0 >= p.n) break;  // warp-uniform
    uint32_t w[32];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      float v[32];
      tmem_ld32(taddr + c2 * 64 + h * 32, v);
      const int cb = c0 + h * 32;
      if (y >= cb && y < cb + 32) {
#pragma unroll
        for (int j = 0; j < 32; ++j)
          if (cb + j == y) zt = v[j] * p.scale;
        hit = true;
      }
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const float ta = v[2 * j] * sc2, tb = v[2 * j + 1] * sc2;
        const bool va = cb + 2 * j < p.n, vb = cb + 2 * j + 1 < p.n;
        const float ea = va ? ex2_sfu(ta - m2) : 0.f;
        const float eb = vb ? ex2_sfu(tb - m2) : 0.f;
        run_s += ea;
        run_e = fmaf(ea, ta, run_e);
        run_s += eb;
        run_e = fmaf(eb, tb, run_e);
        w[h * 16 + j] = pack_bf16x2(ea, eb);
      }
    }
    uint8_t* slot = acquire_slot(slots, slab, lane);
    stage_row128(slot, lane, w);
    flush_slot(tmC, slot, c0, row0, false, lane);
    ++slab;
  }
  if (row_ok) {
    float* q = p.partials + (static_cast<size_t>(row >> 5) * p.nsplit + nb) * kPartialBlock +
               (row & 31);
    q[0] = m2;
    q[32] = run_s;
    q[64] = run_e;
    if (hit) p.ztgt[row] = zt;
  }
}

// ------------------------------------------------------------ the kernel
// Stage geometry.  Solo: one CTA stages A (128 x 64) and B (256 x 64).  Pair:
// the two CTAs of a cluster compute one 256 x 256 tile with a shared
// cta_group::2 MMA; each stages its own 128 rows of A and 128 of the 256 B
// rows, so a stage is 32 KB and seven fit in shared memory (~2 us of MMA
// work buffered against operand latency).
// The G, dW and kept-forward epilogues store through TMA and need 32 KB of staging, so
// their pair-mode ring has six stages.
// WIDE (dH, pair mode): a tile is 256 x 512, two N = 256 MMAs per k-step into
// both TMEM accumulators (so no accumulator double-buffering: at K = V one tile
// is ~1.5 ms of MMA against a few us of epilogue).  Each CTA stages A and two
// B halves, 48 KB a stage, four stages.  Twice the columns per tile halve the
// G row slabs a wave reads from DRAM.
template <bool PAIR, int EPI = EPI_LSE, bool WIDE = false>
struct Geo {
  static constexpr bool kTmaStore = EPI == EPI_GRAD || EPI == EPI_DW || EPI == EPI_LSE_KEEP;
  static constexpr int kHalves = WIDE ? 2 : 1;              // N = 256 MMAs per k-step
  static constexpr int kStages = WIDE ? 4 : (PAIR ? (kTmaStore ? 6 : 7) : 4);
  static constexpr uint32_t kEpiBytes = kTmaStore ? 4 * 2 * kEpiSlotBytes : 0;  // 4 warps x 2 slots
  static constexpr int kBRows = PAIR ? BN / 2 : BN;        // B rows staged per CTA and MMA
  static constexpr uint32_t kABytes = BM * BK * 2;         // 16 KB
  static constexpr uint32_t kBHalfBytes = kBRows * BK * 2;  // 16 or 32 KB
  static constexpr uint32_t kBBytes = kHalves * kBHalfBytes;
  static constexpr uint32_t kStageBytes = kABytes + kBBytes;
  static constexpr int kTileM = PAIR ? 2 * BM : BM;         // output rows per tile
  static constexpr int kTileN = kHalves * BN;               // output columns per tile
  static constexpr size_t kSmem = 1024 + kStages * kStageBytes + kEpiBytes + 512;
  static_assert(!WIDE || (PAIR && (EPI == EPI_DH || EPI == EPI_LSE || EPI == EPI_GRAD)),
                "wide tiles: dH and the logits GEMMs in pair mode only");
  static_assert(kSmem <= 232448, "shared memory per CTA");
};

template <int EPI, bool A_MN, bool B_MN, bool PAIR, bool WIDE = false>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                const __grid_constant__ CUtensorMap tmC, const GemmArgs p) {
  using G = Geo<PAIR, EPI, WIDE>;
  constexpr int S = G::kStages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + S * G::kABytes;
  uint8_t* sEpi = sB + S * G::kBBytes;  // TMA-store staging (1024-byte aligned)
  uint64_t* full_bar = reinterpret_cast<uint64_t*>(sEpi + G::kEpiBytes);
  uint64_t* empty_bar = full_bar + S;
  uint64_t* tfull_bar = empty_bar + S;
  uint64_t* tempty_bar = tfull_bar + 2;
  uint64_t* drain_bar = tempty_bar + 2;
  // Dynamic tile schedule: the leader's producer takes tile ids from a global
  // counter and publishes them through a ring of kRing slots to every other
  // role (the peer CTA's through its own copy of the ring).
  constexpr int kRing = 8;
  uint64_t* ring_full = drain_bar + 1;
  uint64_t* ring_empty = ring_full + kRing;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(ring_empty + kRing);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  volatile int* ring = reinterpret_cast<volatile int*>(tmem_slot + 2);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = PAIR ? cluster_ctarank() : 0u;          // 0 = leader of the pair
  const int unit = PAIR ? static_cast<int>(blockIdx.x >> 1) : static_cast<int>(blockIdx.x);
  const int n_units = PAIR ? static_cast<int>(gridDim.x >> 1) : static_cast<int>(gridDim.x);

  const int M = p.m_count ? clampi(*p.m_count - p.m_offset, 0, p.m_cap) : p.m_static;
  const int K = p.k_count ? clampi(*p.k_count - p.k_offset, 0, p.k_cap) : p.k_static;
  const int mt = (M + G::kTileM - 1) / G::kTileM;
  const int nt = (p.n + G::kTileN - 1) / G::kTileN;
  // Work items.  WIDE: whole tiles for the rounds in which every unit gets
  // one, then the remaining tiles as two 256-column halves each, so the last
  // round is as balanced as with 256 x 256 tiles throughout.
  const int whole = WIDE ? (mt * nt / n_units) * n_units : mt * nt;
  const int num_tiles = WIDE ? whole + 2 * (mt * nt - whole) : mt * nt;
  const int num_kb = (K + BK - 1) / BK;
  const int gm = max(1, p.group_m);
  // item -> tile row, first output column and the N = 256 halves it covers
  auto decode = [&](int item, int& mb, int& col0, int& halves) {
    int tile = item, half = -1;
    if (WIDE && item >= whole) {
      tile = whole + (item - whole) / 2;
      half = (item - whole) & 1;
    }
    int nb;
    tile_coords(tile, mt, nt, gm, p.raster, mb, nb);
    col0 = nb * G::kTileN + (half > 0 ? BN : 0);
    halves = half < 0 ? G::kHalves : 1;
  };
  // dW += (empty chunk): nothing to add.  Uniform across the cluster, before any setup.
  if (EPI == EPI_DW && num_kb == 0 && p.accumulate) return;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull_bar[a], 1);
      mbar_init(&tempty_bar[a], PAIR ? 8 : 4);  // one arrival per epilogue warp of the pair
    }
    mbar_init(drain_bar, 1);
    for (int r = 0; r < kRing; ++r) {
      mbar_init(&ring_full[r], 1);
      // consumers: MMA + 4 epilogue warps (+ the peer's producer and 4 epilogue warps)
      mbar_init(&ring_empty[r], PAIR ? 10 : 5);
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
  }
  if (warp == 1) {
    tmem_alloc<PAIR>(tmem_slot, 2 * BN);
    tmem_relinquish<PAIR>();
  }
  tc_fence_before();
  if (PAIR)
    cluster_sync();  // peer barriers initialised before any remote arrive / TMA signal
  else
    __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const bool dyn = p.tile_counter != nullptr;

  // i-th tile of this CTA (pair) or -1 when done.  Static: unit + i * n_units.
  auto static_tile = [&](int i) { const int t = unit + i * n_units; return t < num_tiles ? t : -1; };
  // Leader producer: take the next tile id and publish it in slot i % kRing.
  auto publish = [&](int i, bool& ok) -> int {
    const int slot = i % kRing;
    if (!mbar_wait(&ring_empty[slot], ((i / kRing) & 1) ^ 1u, abort_flag, p.err, kErrWaitProducer,
                   PAIR)) {
      ok = false;
      return -1;
    }
    int t = atomicAdd(p.tile_counter, 1);
    if (t >= num_tiles) t = -1;
    ring[slot] = t;
    if (PAIR) {
      st_shared_cluster(mapa_shared(smem_u32(const_cast<int*>(&ring[slot])), 1), t);
      mbar_arrive_cluster(mapa_shared(smem_u32(&ring_full[slot]), 1));  // release: orders the store
    }
    mbar_arrive(&ring_full[slot]);
    return t;
  };
  // Any other role (one thread): read slot i % kRing and hand it back.
  auto take = [&](int i, bool& ok, int code) -> int {
    const int slot = i % kRing;
    if (!mbar_wait(&ring_full[slot], (i / kRing) & 1, abort_flag, p.err, code, PAIR)) {
      ok = false;
      return -1;
    }
    const int t = ring[slot];
    if (PAIR)
      mbar_arrive_cluster(mapa_shared(smem_u32(&ring_empty[slot]), 0));  // leader's barrier
    else
      mbar_arrive(&ring_empty[slot]);
    return t;
  };

  if (warp == 0) {
    // ------------------------------------------------ TMA producer (both CTAs)
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int issued = 0;
      bool ok = true;
      // the throttle runs on the pair's leader (the follower's loads feed the same MMAs)
      const bool throttle = p.kprog != nullptr && rank == 0;
      unsigned long long* kstate = reinterpret_cast<unsigned long long*>(p.kprog);
      const int epoch = max(1, p.ksync_epoch);
      long long prog = 0, published = 0;
      // state loaded at the previous check: decided on one epoch later, so the
      // producer never waits for these loads to land
      unsigned long long seen_sum = 0, seen_active = 0;
      for (int i = 0; ok; ++i) {
        const int tile = !dyn ? static_tile(i)
                              : (rank == 0 ? publish(i, ok) : take(i, ok, kErrWaitProducer));
        if (tile < 0) break;
        int mb, col0, halves;
        decode(tile, mb, col0, halves);
        const int a_row = mb * G::kTileM + static_cast<int>(rank) * BM;
        const int b_row = col0 + static_cast<int>(rank) * G::kBRows;  // half h: + h * BN
        const uint32_t tx = PAIR ? 2 * (G::kABytes + halves * G::kBHalfBytes)
                                 : G::kABytes + halves * G::kBHalfBytes;
        for (int kb = 0; kb < num_kb; ++kb) {
          if (throttle && prog % epoch == 0) {
            if (prog == 0) {
              red_add_gpu_u64(kstate + 1, 1ull);  // this unit is running
            } else {
              red_add_gpu_u64(kstate, static_cast<unsigned long long>(prog - published));
              published = prog;
              const long long act = static_cast<long long>(seen_active);
              if (act > 0 && prog * act > static_cast<long long>(seen_sum) +
                                              static_cast<long long>(p.ksync_window) * act)
                ksync_wait(kstate, prog, p.ksync_window);  // ahead a epoch ago: wait on fresh state
            }
            seen_sum = ld_relaxed_gpu_u64(kstate);
            seen_active = ld_relaxed_gpu_u64(kstate + 1);
          }
          ++prog;
          if (!mbar_wait(&empty_bar[stage], phase ^ 1u, abort_flag, p.err, kErrWaitProducer)) {
            ok = false;
            break;
          }
          uint8_t* a_dst = sA + stage * G::kABytes;
          uint8_t* b_dst = sB + stage * G::kBBytes;
          if (!PAIR || rank == 0) mbar_arrive_expect_tx(&full_bar[stage], tx);
          const uint32_t bar = PAIR ? mapa_shared(smem_u32(&full_bar[stage]), 0) : 0u;
          auto load = [&](uint8_t* dst, const CUtensorMap* tm, int x, int y) {
            if (PAIR)
              tma_load_2d_pair(dst, tm, bar, x, y);
            else
              tma_load_2d(dst, tm, &full_bar[stage], x, y);
          };
          if (A_MN) {
#pragma unroll
            for (int j = 0; j < BM / 64; ++j) load(a_dst + j * MN_BLOCK_BYTES, &tmA, a_row + j * 64, kb * BK);
          } else {
            load(a_dst, &tmA, kb * BK, a_row);
          }
          for (int h = 0; h < halves; ++h) {
            uint8_t* bh = b_dst + h * G::kBHalfBytes;
            if (B_MN) {
#pragma unroll
              for (int j = 0; j < G::kBRows / 64; ++j)
                load(bh + j * MN_BLOCK_BYTES, &tmB, b_row + h * BN + j * 64, kb * BK);
            } else {
              load(bh, &tmB, kb * BK, b_row + h * BN);
            }
          }
          ++issued;
          if (++stage == S) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (throttle && prog > 0) {  // done: its progress leaves the running average
        red_add_gpu_u64(kstate, static_cast<unsigned long long>(-published));
        red_add_gpu_u64(kstate + 1, static_cast<unsigned long long>(-1ll));
      }
      if (!ok && (!PAIR || rank == 0)) {
        // Aborted: let the copies already in flight land before the CTA exits.
        int s = stage;
        uint32_t ph = phase;
        for (int i = 0; i < S && i < issued; ++i) {
          if (--s < 0) {
            s = S - 1;
            ph ^= 1u;
          }
          mbar_wait_drain(&full_bar[s], ph);
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer (leader CTA only)
    if (lane == 0 && rank == 0) {
      constexpr uint32_t kIdesc = idesc_bf16_f32(G::kTileM, BN, A_MN, B_MN);
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      if constexpr (WIDE) {
        // Each 256-column half h of the accumulator (TMEM columns h * 256 on)
        // has its own barrier pair tfull / tempty [h].  The last kWideOverlap
        // k-blocks of a tile issue their first-half MMAs first, so the
        // epilogue drains that half while the second-half MMAs finish; the
        // first kWideOverlap k-blocks of the next tile go into the drained
        // first half while the second is drained.  Those k-blocks' stages
        // are freed once both halves have used them.
        uint32_t use0 = 0, use1 = 0;  // tiles that have used each half so far
        auto next = [&](int& st, uint32_t& ph) {
          if (++st == S) {
            st = 0;
            ph ^= 1u;
          }
        };
        auto wait_full = [&](int st, uint32_t ph) {
          if (!mbar_wait(&full_bar[st], ph, abort_flag, p.err, kErrWaitMma)) return false;
          tc_fence_after();
          return true;
        };
        // the four K-steps of stage st into half h
        auto issue_half = [&](int st, int h, int kb) {
          const uint32_t a0 = smem_u32(sA + st * G::kABytes);
          const uint32_t bh = smem_u32(sB + st * G::kBBytes) + h * G::kBHalfBytes;
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            const uint64_t ad = A_MN ? sdesc_sw128(a0 + k * 2048, MN_BLOCK_BYTES, 1024)
                                     : sdesc_sw128(a0 + k * 32, 16, 1024);
            const uint64_t bd = B_MN ? sdesc_sw128(bh + k * 2048, MN_BLOCK_BYTES, 1024)
                                     : sdesc_sw128(bh + k * 32, 16, 1024);
            umma_bf16<PAIR>(tmem_base + static_cast<uint32_t>(h * BN), ad, bd, kIdesc,
                            (kb | k) != 0 ? 1u : 0u);
          }
        };
        auto full_without_mma = [&](int h) {  // K == 0: nothing to wait for
          mbar_arrive(&tfull_bar[h]);
          if (PAIR) mbar_arrive_cluster(mapa_shared(smem_u32(&tfull_bar[h]), 1));
        };
        for (int local = 0; ok; ++local) {
          const int tile = dyn ? take(local, ok, kErrWaitMma) : static_tile(local);
          if (tile < 0) break;
          int mb, col0, halves;
          decode(tile, mb, col0, halves);
          const bool both = halves == 2;
          const int head = both ? min(kWideOverlap, num_kb) : 0;
          const int tail = both ? min(kWideOverlap, num_kb - head) : 0;
          if (!mbar_wait(&tempty_bar[0], (use0 & 1) ^ 1u, abort_flag, p.err, kErrWaitMma)) {
            ok = false;
            break;
          }
          tc_fence_after();
          // head: the first half of the first k-blocks, stages kept
          int st = stage;
          uint32_t ph = phase;
          for (int kb = 0; kb < head; ++kb) {
            if (!wait_full(st, ph)) {
              ok = false;
              break;
            }
            issue_half(st, 0, kb);
            next(st, ph);
          }
          if (!ok) break;
          if (both) {
            if (tail == 0 && num_kb > 0) umma_commit<PAIR>(&tfull_bar[0]);  // first half complete
            if (!mbar_wait(&tempty_bar[1], (use1 & 1) ^ 1u, abort_flag, p.err, kErrWaitMma)) {
              ok = false;
              break;
            }
            tc_fence_after();
            for (int kb = 0; kb < head; ++kb) {  // their second half; then the stages are free
              issue_half(stage, 1, kb);
              umma_commit<PAIR>(&empty_bar[stage]);
              next(stage, phase);
            }
          }
          // both halves (or a half tile's one half) k-block by k-block
          for (int kb = head; kb < num_kb - tail; ++kb) {
            if (!wait_full(stage, phase)) {
              ok = false;
              break;
            }
            issue_half(stage, 0, kb);
            if (both) issue_half(stage, 1, kb);
            umma_commit<PAIR>(&empty_bar[stage]);
            next(stage, phase);
          }
          if (!ok) break;
          if (!both && num_kb > 0) umma_commit<PAIR>(&tfull_bar[0]);
          // tail: the first half of the last k-blocks, then their second half
          st = stage;
          ph = phase;
          for (int kb = num_kb - tail; kb < num_kb; ++kb) {
            if (!wait_full(st, ph)) {
              ok = false;
              break;
            }
            issue_half(st, 0, kb);
            next(st, ph);
          }
          if (!ok) break;
          if (tail > 0) umma_commit<PAIR>(&tfull_bar[0]);
          for (int kb = num_kb - tail; kb < num_kb; ++kb) {
            issue_half(stage, 1, kb);
            umma_commit<PAIR>(&empty_bar[stage]);
            next(stage, phase);
          }
          if (both && num_kb > 0) umma_commit<PAIR>(&tfull_bar[1]);
          if (num_kb == 0) {
            full_without_mma(0);
            if (both) full_without_mma(1);
          }
          ++use0;
          if (both) ++use1;
        }
      } else {
        for (int local = 0;; ++local) {
          const int tile = dyn ? take(local, ok, kErrWaitMma) : static_tile(local);
          if (tile < 0) break;
          // two accumulators used in turn
          const int acc = local & 1;
          const uint32_t acc_phase = (local >> 1) & 1;
          if (!mbar_wait(&tempty_bar[acc], acc_phase ^ 1u, abort_flag, p.err, kErrWaitMma)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * BN);
          for (int kb = 0; kb < num_kb; ++kb) {
            if (!mbar_wait(&full_bar[stage], phase, abort_flag, p.err, kErrWaitMma)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t a0 = smem_u32(sA + stage * G::kABytes);
            const uint32_t b0 = smem_u32(sB + stage * G::kBBytes);
#pragma unroll
            for (int k = 0; k < BK / 16; ++k) {
              const uint64_t ad = A_MN ? sdesc_sw128(a0 + k * 2048, MN_BLOCK_BYTES, 1024)
                                       : sdesc_sw128(a0 + k * 32, 16, 1024);
              const uint64_t bd = B_MN ? sdesc_sw128(b0 + k * 2048, MN_BLOCK_BYTES, 1024)
                                       : sdesc_sw128(b0 + k * 32, 16, 1024);
              umma_bf16<PAIR>(d_tmem, ad, bd, kIdesc, (kb | k) != 0 ? 1u : 0u);
            }
            umma_commit<PAIR>(&empty_bar[stage]);  // frees the stage (in both CTAs) when done
            if (++stage == S) {
              stage = 0;
              phase ^= 1u;
            }
          }
          if (!ok) break;
          if (num_kb > 0) {
            umma_commit<PAIR>(&tfull_bar[acc]);  // accumulator complete (both CTAs)
          } else {                               // K == 0: nothing to wait for
            mbar_arrive(&tfull_bar[acc]);
            if (PAIR) mbar_arrive_cluster(mapa_shared(smem_u32(&tfull_bar[acc]), 1));
          }
        }
      }
      // Every MMA this thread issued must finish before TMEM is released.
      umma_commit_local<PAIR>(drain_bar);
      if (!mbar_wait_drain(drain_bar, 0) && p.err) atomicCAS(p.err, 0, kErrWaitDrain);
    }
  } else {
    // ------------------------------------------------ epilogue warps 2..5 (both CTAs)
    const int q = warp & 3;  // TMEM lanes [32q, 32q+32) are reachable from this warp
    uint8_t* slots = sEpi + (warp - 2) * 2 * kEpiSlotBytes;  // unused unless G::kTmaStore
    int slab = 0;
    uint32_t use0 = 0, use1 = 0;  // WIDE: tiles whose accumulator half 0 / 1 this warp drained
    for (int local = 0;; ++local) {
      int tile;
      if (dyn) {
        bool got = true;
        int t = -1;
        if (lane == 0) t = take(local, got, kErrWaitEpilogue);
        tile = __shfl_sync(0xffffffffu, got ? t : -1, 0);
      } else {
        tile = static_tile(local);
      }
      if (tile < 0) break;
      int mb, col0, halves;
      decode(tile, mb, col0, halves);
      const int row = mb * G::kTileM + static_cast<int>(rank) * BM + q * 32 + lane;
      const int row0 = row - lane;  // first row of this warp
      const uint32_t lanes = tmem_base + (static_cast<uint32_t>(q * 32) << 16);
      // hands accumulator (half) a back to the MMA issuer
      auto release = [&](int a) {
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          if (PAIR)
            mbar_arrive_cluster(mapa_shared(smem_u32(&tempty_bar[a]), 0));  // leader's barrier
          else
            mbar_arrive(&tempty_bar[a]);
        }
      };
      if constexpr (WIDE) {
        // each half as soon as it is complete; a half that starts past the
        // last column has no output (no partials, G or dH columns)
        bool stop = false;
        for (int h = 0; h < halves; ++h) {
          const uint32_t par = (h == 0 ? use0 : use1) & 1u;
          const bool ok = mbar_wait(&tfull_bar[h], par, abort_flag, p.err, kErrWaitEpilogue);
          if (!__all_sync(0xffffffffu, ok)) {
            stop = true;
            break;
          }
          tc_fence_after();
          const int c = col0 + h * BN;
          const uint32_t taddr = lanes + static_cast<uint32_t>(h * BN);
          if (c < p.n) {  // warp-uniform
            if (EPI == EPI_LSE) epi_lse(p, taddr, row, M, c / BN);
            if (EPI == EPI_GRAD) epi_grad_tma(p, &tmC, taddr, row, row0, M, c / BN, slots, slab, lane);
            if (EPI == EPI_DH) epi_dh(p, taddr, row, M, c, BN);
          }
          release(h);
          if (h == 0)
            ++use0;
          else
            ++use1;
        }
        if (stop) break;
      } else {
        const int acc = local & 1;
        const uint32_t acc_phase = (local >> 1) & 1;
        const int nb = col0 / BN;
        const bool ok = mbar_wait(&tfull_bar[acc], acc_phase, abort_flag, p.err, kErrWaitEpilogue);
        if (!__all_sync(0xffffffffu, ok)) break;
        tc_fence_after();
        const uint32_t taddr = lanes + static_cast<uint32_t>(acc * BN);
        if (EPI == EPI_LSE) epi_lse(p, taddr, row, M, nb);
        if (EPI == EPI_GRAD) epi_grad_tma(p, &tmC, taddr, row, row0, M, nb, slots, slab, lane);
        if (EPI == EPI_LSE_KEEP) epi_lse_keep(p, &tmC, taddr, row, row0, M, nb, slots, slab, lane);
        if (EPI == EPI_DH) epi_dh(p, taddr, row, M, col0, BN);
        if (EPI == EPI_DW) epi_dw_tma(p, &tmC, taddr, row0, nb, num_kb == 0, slots, slab, lane);
        release(acc);
      }
    }
    if (G::kTmaStore) {
      if (lane == 0) bulk_wait_all();  // stores complete before the CTA exits
      __syncwarp();
    }
  }

  tc_fence_before();
  __syncwarp();
  if (PAIR)
    cluster_sync();  // no CTA leaves while its pair may still touch its smem or TMEM
  else
    __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc<PAIR>(tmem_base, 2 * BN);
  }
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  // looked up once (a function-local static: initialised once, thread-safe)
  static const EncodeTiledFn fn = [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    return cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                            &q) == cudaSuccess &&
                   q == cudaDriverEntryPointSuccess
               ? reinterpret_cast<EncodeTiledFn>(ptr)
               : nullptr;
  }();
  return fn;
}

template <int EPI, bool A_MN, bool B_MN, bool PAIR, bool WIDE = false>
cudaError_t launch_one(const CUtensorMap& ta, const CUtensorMap& tb, const CUtensorMap& tc,
                       const GemmArgs& args, int grid, cudaStream_t s) {
  auto k = gemm_kernel<EPI, A_MN, B_MN, PAIR, WIDE>;
  const size_t smem = Geo<PAIR, EPI, WIDE>::kSmem;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(grid), 1, 1);
  cfg.blockDim = dim3(NUM_THREADS, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = PAIR ? 2 : 1;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, k, ta, tb, tc, args);
  note_launches(1);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace

size_t gemm_smem_bytes(bool pair) { return pair ? Geo<true, EPI_GRAD>::kSmem : Geo<false, EPI_GRAD>::kSmem; }

int gemm_tile_m(bool pair) { return pair ? Geo<true>::kTileM : Geo<false>::kTileM; }

int gemm_b_box_rows(bool pair) { return pair ? Geo<true>::kBRows : Geo<false>::kBRows; }

namespace {
cudaError_t make_tmap_2d(CUtensorMap* tm, CUtensorMapDataType type, const void* base, uint64_t inner,
                         uint64_t outer, uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return cudaErrorNotSupported;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {row_bytes};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(tm, type, 2, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}
}  // namespace

cudaError_t make_tmap_bf16(CUtensorMap* tm, const void* base, uint64_t inner, uint64_t outer,
                           uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer) {
  return make_tmap_2d(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, base, inner, outer, row_bytes, box_inner,
                      box_outer);
}

cudaError_t make_tmap_f32(CUtensorMap* tm, const void* base, uint64_t inner, uint64_t outer,
                          uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer) {
  return make_tmap_2d(tm, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, base, inner, outer, row_bytes, box_inner,
                      box_outer);
}

namespace {
// One thread waits, through the kernels' own bounded wait, on an mbarrier that
// nothing arrives on: the wait gives up after kWaitTimeoutNs and records
// kErrWaitSelftest in the error word, and the kernel returns.
__global__ void bounded_wait_selftest_kernel(int* err) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  abort_flag = 0;
  mbar_init(&bar, 1);
  mbar_wait(&bar, 0, &abort_flag, err, kErrWaitSelftest);
}
}  // namespace

cudaError_t launch_bounded_wait_selftest(int* err, cudaStream_t s) {
  bounded_wait_selftest_kernel<<<1, 1, 0, s>>>(err);
  note_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_gemm(int epi, bool a_mn, bool b_mn, bool pair, const CUtensorMap& ta,
                        const CUtensorMap& tb, const CUtensorMap& tc, const GemmArgs& args, int grid,
                        cudaStream_t s, bool wide) {
  if (wide && pair && epi == EPI_DH && !a_mn && b_mn)
    return launch_one<EPI_DH, false, true, true, true>(ta, tb, tc, args, grid, s);
  if (wide && pair && epi == EPI_LSE && !a_mn && !b_mn)
    return launch_one<EPI_LSE, false, false, true, true>(ta, tb, tc, args, grid, s);
  if (wide && pair && epi == EPI_GRAD && !a_mn && !b_mn)
    return launch_one<EPI_GRAD, false, false, true, true>(ta, tb, tc, args, grid, s);
#define SPO_GEMM_CASE(E, AM, BMN)                                                        \
  if (epi == E && a_mn == AM && b_mn == BMN)                                             \
    return pair ? launch_one<E, AM, BMN, true>(ta, tb, tc, args, grid, s)                \
                : launch_one<E, AM, BMN, false>(ta, tb, tc, args, grid, s);
  SPO_GEMM_CASE(EPI_LSE, false, false)
  SPO_GEMM_CASE(EPI_LSE_KEEP, false, false)
  SPO_GEMM_CASE(EPI_GRAD, false, false)
  SPO_GEMM_CASE(EPI_DH, false, true)
  SPO_GEMM_CASE(EPI_DW, true, true)
#undef SPO_GEMM_CASE
  return cudaErrorInvalidValue;
}

}  // namespace spo
