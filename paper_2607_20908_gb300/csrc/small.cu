// small.cu -- the bandwidth- and latency-bound steps of the path: loss-token
// selection, row compaction and gather, the split-vocabulary logsumexp
// combine, group-normalised advantages and the policy-loss forward.
#include <math.h>

#include <atomic>

#include "internal.h"

namespace spo {

namespace {

constexpr int kCompactThreads = 256;
constexpr int kCompactItems = 4;
constexpr int kCompactTile = kCompactThreads * kCompactItems;  // tokens per block
constexpr float kLn2 = 0.69314718055994531f;
constexpr float kLog2e = 1.4426950408889634f;

__device__ __forceinline__ bool selected(int kind, const uint8_t* mask, const int* tgt,
                                         const float* g, long long t) {
  if (kind == 0) return (mask == nullptr || mask[t] != 0) && tgt[t] >= 0;
  return g[t] != 0.f;
}

// Exclusive block-wide prefix sum of one int per thread (blockDim = 256).
__device__ __forceinline__ int block_exclusive_scan(int v, int* total) {
  __shared__ int warp_sums[kCompactThreads / 32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_sums[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int w = lane < kCompactThreads / 32 ? warp_sums[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    if (lane < kCompactThreads / 32) warp_sums[lane] = w;
  }
  __syncthreads();
  const int before = (warp > 0 ? warp_sums[warp - 1] : 0) + x - v;
  if (total) *total = warp_sums[kCompactThreads / 32 - 1];
  __syncthreads();
  return before;
}

__global__ void compact_count_kernel(int kind, const uint8_t* mask, const int* tgt, const float* g,
                                     long long T, int* block_counts) {
  const long long base = static_cast<long long>(blockIdx.x) * kCompactTile;
  int c = 0;
#pragma unroll
  for (int i = 0; i < kCompactItems; ++i) {
    const long long t = base + static_cast<long long>(threadIdx.x) * kCompactItems + i;
    if (t < T && selected(kind, mask, tgt, g, t)) ++c;
  }
  int total;
  block_exclusive_scan(c, &total);
  if (threadIdx.x == 0) block_counts[blockIdx.x] = total;
}

// Single block: exclusive scan of the per-block counts, total -> *count.
__global__ void compact_scan_kernel(const int* block_counts, int nblocks, int* block_offsets,
                                    int* count) {
  __shared__ int carry;
  if (threadIdx.x == 0) carry = 0;
  __syncthreads();
  for (int base = 0; base < nblocks; base += kCompactThreads) {
    const int i = base + threadIdx.x;
    const int v = i < nblocks ? block_counts[i] : 0;
    int total;
    const int ex = block_exclusive_scan(v, &total);
    if (i < nblocks) block_offsets[i] = carry + ex;
    __syncthreads();
    if (threadIdx.x == 0) carry += total;
    __syncthreads();
  }
  if (threadIdx.x == 0) *count = carry;
}

__global__ void compact_write_kernel(int kind, const uint8_t* mask, const int* tgt, const float* g,
                                     long long T, const int* block_offsets, int* idx) {
  const long long base = static_cast<long long>(blockIdx.x) * kCompactTile;
  bool f[kCompactItems];
  int c = 0;
#pragma unroll
  for (int i = 0; i < kCompactItems; ++i) {
    const long long t = base + static_cast<long long>(threadIdx.x) * kCompactItems + i;
    f[i] = t < T && selected(kind, mask, tgt, g, t);
    c += f[i];
  }
  int pos = block_offsets[blockIdx.x] + block_exclusive_scan(c, nullptr);
#pragma unroll
  for (int i = 0; i < kCompactItems; ++i) {
    if (f[i]) idx[pos++] = static_cast<int>(base + static_cast<long long>(threadIdx.x) * kCompactItems + i);
  }
}

// One warp per compacted row: copy the bf16 row in 16-byte pieces.
__global__ void gather_kernel(const uint4* H, int row_vecs, const int* idx, const int* count,
                              int rows_cap, uint4* Hc, const int* tgt, int* tgt_c,
                              long long tgt_off, long long tgt_lim, const float* a, float* a_c,
                              const float* b, float* b_c) {
  const int n = *count;
  const int zero_end = min(rows_cap, (n + kRowPad - 1) / kRowPad * kRowPad);
  const int warps_per_block = blockDim.x >> 5;
  const int lane = threadIdx.x & 31;
  for (int r = blockIdx.x * warps_per_block + (threadIdx.x >> 5); r < zero_end;
       r += gridDim.x * warps_per_block) {
    uint4* dst = Hc + static_cast<size_t>(r) * row_vecs;
    if (r < n) {
      const int src_row = idx[r];
      const uint4* src = H + static_cast<size_t>(src_row) * row_vecs;
      for (int i = lane; i < row_vecs; i += 32) dst[i] = src[i];
      if (lane == 0) {
        if (tgt_c) {
          const long long y = static_cast<long long>(tgt[src_row]) - tgt_off;
          tgt_c[r] = (y >= 0 && y < tgt_lim) ? static_cast<int>(y) : -1;
        }
        if (a_c) a_c[r] = a[src_row];
        if (b_c) b_c[r] = b[src_row];
      }
    } else {
      for (int i = lane; i < row_vecs; i += 32) dst[i] = make_uint4(0, 0, 0, 0);
      if (lane == 0) {
        if (tgt_c) tgt_c[r] = 0;
        if (a_c) a_c[r] = 0.f;
        if (b_c) b_c[r] = 0.f;
      }
    }
  }
}

// Merge (m2, s2, e2) into (m, s, e); m in log2 units, s = sum 2^(t-m), e = sum 2^(t-m) t.
// One exponential: the side with the smaller max is rescaled onto the larger.
__device__ __forceinline__ void lse_merge(float& m, float& s, float& e, float m2, float s2, float e2) {
  if (m2 == -INFINITY) return;
  if (m2 <= m) {
    const float r = exp2f(m2 - m);
    s = fmaf(s2, r, s);
    e = fmaf(e2, r, e);
  } else {
    const float r = exp2f(m - m2);  // m = -inf gives r = 0
    s = fmaf(s, r, s2);
    e = fmaf(e, r, e2);
    m = m2;
  }
}

constexpr int kCombineRows = 16;   // rows per block: 1024 blocks at T = 16384 balance 152 SMs
constexpr int kCombineGroups = 16; // split groups per row (8 warps x 2 half-warps)
constexpr int kCombineUnroll = 4;  // vocab tiles whose loads a thread has in flight at once

// Split-vocabulary combine.  A block owns 16 rows; half-warp h of warp w
// merges vocab tiles 2w + h, 2w + h + 16, ... of those rows in ascending
// order (each load is a contiguous 64-byte run of one plane of the
// row-block-major partials), and the 16 per-group results are merged through
// shared memory.  The partials are read once, so the loads stream past L1/L2.
__global__ void __launch_bounds__(256) lse_combine_kernel(const float* partials, int nsplit,
                                                          const float* ztgt, const int* idx,
                                                          const int* count, float* logp,
                                                          float* entropy, float* lse_out,
                                                          const int* tgt_c, float4* rec) {
  __shared__ float sm[kCombineGroups][kCombineRows][3];
  const int n = *count;
  const int row0 = blockIdx.x * kCombineRows;
  if (row0 >= n) return;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int r = lane & 15, grp = warp * 2 + (lane >> 4);
  const int row = row0 + r;
  float m = -INFINITY, s = 0.f, e = 0.f;
  if (row < n) {
    const float* slab = partials + static_cast<size_t>(row >> 5) * nsplit * kPartialBlock + (row & 31);
    int j = grp;
    for (; j + (kCombineUnroll - 1) * kCombineGroups < nsplit; j += kCombineUnroll * kCombineGroups) {
      float pm[kCombineUnroll], ps[kCombineUnroll], pe[kCombineUnroll];
#pragma unroll
      for (int u = 0; u < kCombineUnroll; ++u) {
        const float* q = slab + static_cast<size_t>(j + u * kCombineGroups) * kPartialBlock;
        pm[u] = __ldcs(q);
        ps[u] = __ldcs(q + 32);
        pe[u] = __ldcs(q + 64);
      }
#pragma unroll
      for (int u = 0; u < kCombineUnroll; ++u) lse_merge(m, s, e, pm[u], ps[u], pe[u]);
    }
    for (; j < nsplit; j += kCombineGroups) {
      const float* q = slab + static_cast<size_t>(j) * kPartialBlock;
      lse_merge(m, s, e, __ldcs(q), __ldcs(q + 32), __ldcs(q + 64));
    }
  }
  sm[grp][r][0] = m;
  sm[grp][r][1] = s;
  sm[grp][r][2] = e;
  __syncthreads();
  if (threadIdx.x < kCombineRows && row0 + static_cast<int>(threadIdx.x) < n) {
    const int rr = threadIdx.x;
    float M = sm[0][rr][0], S = sm[0][rr][1], E = sm[0][rr][2];
    for (int g = 1; g < kCombineGroups; ++g) lse_merge(M, S, E, sm[g][rr][0], sm[g][rr][1], sm[g][rr][2]);
    const int crow = row0 + rr;
    const int t = idx[crow];
    if (rec) {  // one vocabulary slice: hand the merged partial on
      rec[t] = make_float4(M, S, E, tgt_c[crow] >= 0 ? ztgt[crow] : -INFINITY);
      return;
    }
    const float lse2 = M + log2f(S);
    const float lse_nat = lse2 * kLn2;
    logp[t] = ztgt[crow] - lse_nat;
    if (entropy) entropy[t] = (lse2 - E / S) * kLn2;
    if (lse_out) lse_out[t] = lse_nat;
  }
}

// Merge of the vocabulary slices' records: one thread per token, slices in
// ascending order.  The target logit is the one finite z_tgt among them.
__global__ void merge_slices_kernel(const float4* rec, int n_slices, long long T, float* logp,
                                    float* entropy, float* lse_out) {
  const long long t = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (t >= T) return;
  float m = -INFINITY, s = 0.f, e = 0.f, zt = -INFINITY;
  for (int k = 0; k < n_slices; ++k) {
    const float4 q = rec[static_cast<long long>(k) * T + t];
    if (q.y > 0.f) {
      lse_merge(m, s, e, q.x, q.y, q.z);
      zt = fmaxf(zt, q.w);
    }
  }
  if (s > 0.f) {
    const float lse2 = m + log2f(s);
    const float lse_nat = lse2 * kLn2;
    logp[t] = zt - lse_nat;
    if (entropy) entropy[t] = (lse2 - e / s) * kLn2;
    if (lse_out) lse_out[t] = lse_nat;
  } else {
    logp[t] = 0.f;
    if (entropy) entropy[t] = 0.f;
    if (lse_out) lse_out[t] = 0.f;
  }
}

// G from the kept forward, in place: for compacted row r < count and column v,
//   G = inv_temp * g_t * (1[v == y_t] - E[r, v] * 2^(m[r, v / 256] - lse_t log2 e))
// with E = 2^(t - m) kept by the forward and m its per-tile max (log2 units,
// the partials' first plane).  Eight bf16 per thread (16-byte accesses).
__global__ void form_g_kernel(__nv_bfloat16* E, long long ldE, int V, const float* partials,
                              int nsplit, const int* idx, const int* count, const int* tgt_c,
                              const float* lse, const float* g, float inv_temp) {
  const int n = *count;
  const int vec = V / 8;
  const long long total = static_cast<long long>(n) * vec;
  for (long long k = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; k < total;
       k += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int r = static_cast<int>(k / vec);
    const int v0 = static_cast<int>(k - static_cast<long long>(r) * vec) * 8;
    const int t = idx[r];
    const float coef = inv_temp * g[t];
    const int y = tgt_c[r];
    const float m = partials[(static_cast<size_t>(r >> 5) * nsplit + (v0 >> 8)) * kPartialBlock +
                             (r & 31)];
    const float scale = exp2f(m - lse[t] * kLog2e);   // 2^(m - lse log2 e)
    uint4* p = reinterpret_cast<uint4*>(E + static_cast<size_t>(r) * ldE + v0);
    uint4 w = *p;
    __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&w);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float2 e = __bfloat1622float2(h[j]);
      const int va = v0 + 2 * j;
      const float ga = coef * ((va == y ? 1.f : 0.f) - e.x * scale);
      const float gb = coef * ((va + 1 == y ? 1.f : 0.f) - e.y * scale);
      h[j] = __floats2bfloat162_rn(ga, gb);
    }
    *p = w;
  }
}

// One warp per sequence: ballot + popcount prefix over its tokens.
__global__ void token_select_kernel(const int* cu, const uint8_t* mask, const int* tgt, int n_seq,
                                    int window, uint8_t* loss_mask, int* n_tok) {
  const int warps = blockDim.x >> 5;
  const int seq = blockIdx.x * warps + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (seq >= n_seq) return;
  const int b = cu[seq], e = cu[seq + 1];
  int kept = 0;
  for (int base = b; base < e; base += 32) {
    const int t = base + lane;
    const bool in = t < e;
    const bool elig = in && (mask == nullptr || mask[t] != 0) && tgt[t] >= 0;
    const unsigned bal = __ballot_sync(0xffffffffu, elig);
    const int rank = kept + __popc(bal & ((1u << lane) - 1u));
    if (in) loss_mask[t] = (elig && (window <= 0 || rank < window)) ? 1 : 0;
    kept += __popc(bal);
  }
  if (lane == 0) n_tok[seq] = (window > 0 && kept > window) ? window : kept;
}

// Group-normalised advantages of one group g, computed by one warp.  The
// members are the indices i in [b, e) (with gid[i] == g when check_gid) and
// are visited in ascending index; every operation is a single IEEE fp32
// operation in a fixed order, so the result is reproducible bit for bit (the
// _rn intrinsics also keep the compiler from contracting into fused
// multiply-adds).
__device__ __forceinline__ void group_adv_warp(const float* rewards, const int* gid, int g, int b,
                                               int e, bool check_gid, int std_mode, float eps,
                                               float* adv, int lane) {
  float acc = 0.f, lo = INFINITY, hi = -INFINITY;
  int n = 0;
  for (int base = b; base < e; base += 32) {
    const int i = base + lane;
    const bool mem = i < e && (!check_gid || gid[i] == g);
    const float r = mem ? rewards[i] : 0.f;
    unsigned bal = __ballot_sync(0xffffffffu, mem);
    while (bal) {
      const int l = __ffs(bal) - 1;
      const float rl = __shfl_sync(0xffffffffu, r, l);
      acc = __fadd_rn(acc, rl);
      lo = fminf(lo, rl);
      hi = fmaxf(hi, rl);
      ++n;
      bal &= bal - 1u;
    }
  }
  const bool zero = n <= 1 || lo == hi;
  float mu = 0.f, den = 1.f;
  if (!zero) {
    mu = __fdiv_rn(acc, static_cast<float>(n));
    float ss = 0.f;
    for (int base = b; base < e; base += 32) {
      const int i = base + lane;
      const bool mem = i < e && (!check_gid || gid[i] == g);
      const float dv = mem ? __fsub_rn(rewards[i], mu) : 0.f;
      unsigned bal = __ballot_sync(0xffffffffu, mem);
      while (bal) {
        const int l = __ffs(bal) - 1;
        const float dl = __shfl_sync(0xffffffffu, dv, l);
        ss = __fadd_rn(ss, __fmul_rn(dl, dl));
        bal &= bal - 1u;
      }
    }
    const float var = __fdiv_rn(ss, static_cast<float>(std_mode == 0 ? n - 1 : n));
    den = __fadd_rn(__fsqrt_rn(var), eps);
  }
  for (int base = b; base < e; base += 32) {
    const int i = base + lane;
    if (i < e && (!check_gid || gid[i] == g))
      adv[i] = zero ? 0.f : __fdiv_rn(__fsub_rn(rewards[i], mu), den);
  }
}

// One warp per group, scanning every sequence: O(n_groups * n_seq) reads, no
// scratch memory; the right shape for the few hundred sequences of a step.
__global__ void group_adv_kernel(const float* rewards, const int* gid, int n_seq, int n_groups,
                                 int std_mode, float eps, float* adv) {
  const int warps = blockDim.x >> 5;
  const int g = blockIdx.x * warps + (threadIdx.x >> 5);
  if (g >= n_groups) return;
  group_adv_warp(rewards, gid, g, 0, n_seq, true, std_mode, eps, adv, threadIdx.x & 31);
}

// Runs of equal group ids: the number of runs of each group and the start /
// end of its run (meaningful when it has one).  The atomics' results are not
// waited for.
__global__ void adv_runs_kernel(const int* gid, int n_seq, int n_groups, int* runs, int* start,
                                int* end) {
  const int stride = gridDim.x * blockDim.x;
  for (int i0 = blockIdx.x * blockDim.x + threadIdx.x; i0 < n_seq; i0 += 4 * stride) {
    int gv[4], gp[4], gn[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {  // the loads of four elements in flight together
      const int i = i0 + u * stride;
      gv[u] = i < n_seq ? gid[i] : -1;
      gp[u] = i < n_seq && i > 0 ? gid[i - 1] : -1;
      gn[u] = i + 1 < n_seq ? gid[i + 1] : -1;
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int i = i0 + u * stride;
      const int g = gv[u];
      if (i >= n_seq || g < 0 || g >= n_groups) continue;  // no group: no advantage
      if (i == 0 || gp[u] != g) {
        atomicAdd(&runs[g], 1);
        start[g] = i;
      }
      if (i == n_seq - 1 || gn[u] != g) end[g] = i + 1;
    }
  }
}

// Raises *split when some group has more than one run (its members are not
// contiguous).
__global__ void adv_split_kernel(const int* runs, int n_groups, int* split) {
  bool multi = false;
  for (int g = blockIdx.x * blockDim.x + threadIdx.x; g < n_groups; g += gridDim.x * blockDim.x)
    multi |= runs[g] > 1;
  if (__any_sync(0xffffffffu, multi) && (threadIdx.x & 31) == 0) atomicOr(split, 1);
}

// The same fold by one thread over a contiguous run [b, e): the identical
// sequence of fp32 operations, without the warp's shuffles, so a warp
// handles 32 groups at once.  Element i lives at src[at(i)] and its advantage
// goes to dst[at(i)].
template <class At>
__device__ __forceinline__ void group_adv_thread(const float* src, int b, int e, int std_mode,
                                                 float eps, float* dst, At at) {
  constexpr int kB = 8;  // loads issued before the fold consumes them
  float acc = 0.f, lo = INFINITY, hi = -INFINITY;
  for (int i0 = b; i0 < e; i0 += kB) {
    float r[kB];
#pragma unroll
    for (int u = 0; u < kB; ++u) r[u] = i0 + u < e ? src[at(i0 + u)] : 0.f;
#pragma unroll
    for (int u = 0; u < kB; ++u) {
      if (i0 + u < e) {
        acc = __fadd_rn(acc, r[u]);
        lo = fminf(lo, r[u]);
        hi = fmaxf(hi, r[u]);
      }
    }
  }
  const int n = e - b;
  const bool zero = n <= 1 || lo == hi;
  float mu = 0.f, den = 1.f;
  if (!zero) {
    mu = __fdiv_rn(acc, static_cast<float>(n));
    float ss = 0.f;
    for (int i0 = b; i0 < e; i0 += kB) {
      float r[kB];
#pragma unroll
      for (int u = 0; u < kB; ++u) r[u] = i0 + u < e ? src[at(i0 + u)] : 0.f;
#pragma unroll
      for (int u = 0; u < kB; ++u) {
        if (i0 + u < e) {
          const float dv = __fsub_rn(r[u], mu);
          ss = __fadd_rn(ss, __fmul_rn(dv, dv));
        }
      }
    }
    const float var = __fdiv_rn(ss, static_cast<float>(std_mode == 0 ? n - 1 : n));
    den = __fadd_rn(__fsqrt_rn(var), eps);
  }
  for (int i = b; i < e; ++i)
    dst[at(i)] = zero ? 0.f : __fdiv_rn(__fsub_rn(src[at(i)], mu), den);
}

struct AtIdentity {
  __device__ int operator()(int i) const { return i; }
};
// one pad word per 32: consecutive threads' runs fall in different banks
struct AtPadded {
  __device__ int operator()(int i) const { return i + (i >> 5); }
};

// Second pass of the run path.  When every group is one run, a block takes 256
// consecutive group ids; if their runs lie back to back in memory (the usual
// packing) and span at most kAdvStage rewards, the block stages that span in
// shared memory with coalesced loads, each thread folds its own group there,
// and the advantages go back with coalesced stores.  Other blocks fold each
// group straight from memory, one thread per group.  When some group has
// several runs, one warp per group scans every sequence.  In every case the
// members are folded in ascending index: the same bits.
constexpr int kAdvStage = 8192;

__global__ void __launch_bounds__(256) group_adv_runs_kernel(
    const float* rewards, const int* gid, int n_seq, int n_groups, int std_mode, float eps,
    const int* runs, const int* start, const int* end, const int* split, float* adv) {
  __shared__ float st[kAdvStage + kAdvStage / 32];
  if (*split) {
    const int lane = threadIdx.x & 31;
    const int warps = (gridDim.x * blockDim.x) >> 5;
    for (int g = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; g < n_groups; g += warps)
      group_adv_warp(rewards, gid, g, 0, n_seq, true, std_mode, eps, adv, lane);
    return;
  }
  for (int g0 = blockIdx.x * blockDim.x; g0 < n_groups; g0 += gridDim.x * blockDim.x) {
    const int g = g0 + threadIdx.x;
    const bool live = g < n_groups;
    const int b = live && runs[g] > 0 ? start[g] : 0;
    const int e = live && runs[g] > 0 ? end[g] : 0;
    // back to back: every group of the block non-empty, each run starting where
    // the previous group's ends
    const int g_last = min(n_groups, g0 + static_cast<int>(blockDim.x)) - 1;
    const int lo = runs[g0] > 0 ? start[g0] : 0;
    const int hi = runs[g_last] > 0 ? end[g_last] : 0;
    const bool chained =
        !live || (runs[g] > 0 && (g == g0 || (runs[g - 1] > 0 && end[g - 1] == b)));
    const bool staged = __syncthreads_and(chained) && hi - lo > 0 && hi - lo <= kAdvStage;
    if (!staged) {
      if (live && e > b) group_adv_thread(rewards, b, e, std_mode, eps, adv, AtIdentity());
      continue;
    }
    const AtPadded at;
    for (int k = threadIdx.x; k < hi - lo; k += blockDim.x) st[at(k)] = rewards[lo + k];
    __syncthreads();
    if (live) group_adv_thread(st, b - lo, e - lo, std_mode, eps, st, at);
    __syncthreads();
    for (int k = threadIdx.x; k < hi - lo; k += blockDim.x) adv[lo + k] = st[at(k)];
    __syncthreads();
  }
}

// Composite reward of one candidate: the piecewise verifiable reward
// (compile penalty; correctness penalty; clipped log2 speedup and stability
// penalty once every test passes) plus the structural score.
__device__ __forceinline__ float composite_reward(uint8_t compiled, float p, float speedup, float cv,
                                                  float r_struct, const RewardParams& q) {
  float r;
  if (compiled == 0) {
    r = -q.alpha_comp;
  } else {
    r = -q.alpha_wrong * (1.f - p);
    if (p >= 1.f) {
      const float ls = speedup > 0.f ? log2f(speedup) : -INFINITY;  // no usable speedup: lower bound
      r += q.alpha_speed * fminf(fmaxf(ls, q.s_min), q.s_max);
      r += -q.alpha_cv * cv;
    }
  }
  return r + r_struct;
}

__global__ void reward_kernel(const uint8_t* compiled, const float* pass_rate, const float* speedup,
                              const float* cv, const float* r_struct, int n, RewardParams q,
                              float* out) {
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x)
    out[i] = composite_reward(compiled[i], pass_rate[i], speedup[i], cv[i],
                              r_struct ? r_struct[i] : 0.f, q);
}

// Same, four candidates per thread with 16-byte loads (all operands aligned).
__global__ void reward_kernel_x4(const uchar4* compiled, const float4* pass_rate,
                                 const float4* speedup, const float4* cv, const float4* r_struct,
                                 int n4, RewardParams q, float4* out) {
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += gridDim.x * blockDim.x) {
    const uchar4 c = compiled[i];
    const float4 p = pass_rate[i], s = speedup[i], v = cv[i];
    const float4 r = r_struct ? r_struct[i] : make_float4(0.f, 0.f, 0.f, 0.f);
    out[i] = make_float4(composite_reward(c.x, p.x, s.x, v.x, r.x, q),
                         composite_reward(c.y, p.y, s.y, v.y, r.y, q),
                         composite_reward(c.z, p.z, s.z, v.z, r.z, q),
                         composite_reward(c.w, p.w, s.w, v.w, r.w, q));
  }
}

__global__ void scale_kernel(float* x, long long n, float alpha, const float* alpha_dev) {
  const float a = alpha_dev ? *alpha_dev : alpha;
  for (long long i = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<long long>(gridDim.x) * blockDim.x)
    x[i] *= a;
}

// Input validation: one grid-stride pass, integer atomics (counts are exact).
__global__ void validate_kernel(const int* tgt, long long T, long long V, const int* cu, int n_seq,
                                const int* gid, int n_groups, const float* rewards,
                                const float* old_logp, const float* ref_logp, const uint8_t* mask,
                                int* counts) {
  int c[6] = {0, 0, 0, 0, 0, 0};
  const long long stride = static_cast<long long>(gridDim.x) * blockDim.x;
  const long long i0 = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x;
  for (long long t = i0; t < T; t += stride) {
    if (tgt && tgt[t] >= V) ++c[0];
    if (old_logp && !isfinite(old_logp[t])) ++c[4];
    if (ref_logp && !isfinite(ref_logp[t])) ++c[4];
    if (mask && mask[t] > 1) ++c[5];
  }
  for (long long i = i0; i < n_seq; i += stride) {
    if (cu && cu[i + 1] < cu[i]) ++c[1];
    if (gid && (gid[i] < 0 || gid[i] >= n_groups)) ++c[2];
    if (rewards && !isfinite(rewards[i])) ++c[3];
  }
  if (i0 == 0 && cu) c[1] += (cu[0] != 0) + (cu[n_seq] != T);
#pragma unroll
  for (int k = 0; k < 6; ++k)
    if (c[k]) atomicAdd(&counts[k], c[k]);
}

// ---------------------------------------------------------------- policy loss
constexpr int kLossThreads = 256;

__device__ __forceinline__ double block_sum_d(double v, double* sh) {
  // fixed-order tree over the block (deterministic for a fixed blockDim)
  sh[threadIdx.x] = v;
  __syncthreads();
  for (int s = kLossThreads / 2; s > 0; s >>= 1) {
    if (threadIdx.x < s) sh[threadIdx.x] += sh[threadIdx.x + s];
    __syncthreads();
  }
  const double r = sh[0];
  __syncthreads();
  return r;
}

// One warp per sequence; the grid strides over sequences.
__device__ __forceinline__ int warp_seq0() { return (blockIdx.x * blockDim.x + threadIdx.x) >> 5; }
__device__ __forceinline__ int warp_seq_stride() { return (gridDim.x * blockDim.x) >> 5; }

// Sum over a warp by a fixed xor butterfly: every lane ends with the same bits.
__device__ __forceinline__ float warp_sum_f(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = __fadd_rn(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ long long warp_sum_ll(long long v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// (a) loss tokens per sequence and sequences per group (integers).
__global__ void loss_count_kernel(const int* cu, const int* gid, const uint8_t* lm, int n_seq,
                                  int n_groups, int* n_tok, int* gsize) {
  const int lane = threadIdx.x & 31;
  for (int i = warp_seq0(); i < n_seq; i += warp_seq_stride()) {
    const int b = cu[i], e = cu[i + 1];
    int c = 0;
    for (int t0 = b + lane; t0 < e; t0 += 128) {
      uint8_t m[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) m[u] = t0 + 32 * u < e ? lm[t0 + 32 * u] : 0;
#pragma unroll
      for (int u = 0; u < 4; ++u) c += m[u] ? 1 : 0;
    }
    c = __reduce_add_sync(0xffffffffu, c);
    if (lane == 0) {
      n_tok[i] = c;
      const int g = gid[i];
      if (g >= 0 && g < n_groups) atomicAdd(&gsize[g], 1);
    }
  }
}

// (b) number of non-empty groups and of loss tokens (integer sums; scal zeroed).
__global__ void loss_scalars_kernel(const int* gsize, int n_groups, const int* n_tok, int n_seq,
                                    unsigned long long* scal) {
  long long ng = 0, nt = 0;
  for (int k = blockIdx.x * blockDim.x + threadIdx.x; k < max(n_groups, n_seq);
       k += gridDim.x * blockDim.x) {
    if (k < n_groups) ng += gsize[k] > 0 ? 1 : 0;
    if (k < n_seq) nt += n_tok[k];
  }
  ng = warp_sum_ll(ng);
  nt = warp_sum_ll(nt);
  if ((threadIdx.x & 31) == 0) {
    if (ng) atomicAdd(&scal[0], static_cast<unsigned long long>(ng));
    if (nt) atomicAdd(&scal[1], static_cast<unsigned long long>(nt));
  }
}

// (c) per-token surrogate, KL, dL/dlogp; per-sequence fp64 partial sums (each
// lane over tokens b + lane, b + lane + 32, ..., then the fixed butterfly).
__global__ void loss_token_kernel(const float* logp, const float* old_logp, const float* ref_logp,
                                  const float* adv, const int* cu, const int* gid, int n_seq,
                                  int n_groups, const uint8_t* lm, float clip_eps, float kl_beta,
                                  int agg, const int* n_tok, const int* gsize,
                                  const unsigned long long* scal, float* g, double* part,
                                  int* part_clip) {
  const int lane = threadIdx.x & 31;
  const bool use_kl = ref_logp != nullptr && kl_beta != 0.f;
  const float lo = 1.f - clip_eps, hi = 1.f + clip_eps;
  for (int i = warp_seq0(); i < n_seq; i += warp_seq_stride()) {
    const int b = cu[i], e = cu[i + 1];
    const int ni = n_tok[i];
    // c_t of Eq. 3's average; fp32 (GB300's fp64 unit is narrow, and every
    // lane of the warp computes it)
    float c = 0.f;
    if (agg == 0) {
      const unsigned long long ng = scal[0];
      const int gi = gid[i];
      if (ni > 0 && ng > 0 && gi >= 0 && gi < n_groups)
        c = __frcp_rn(static_cast<float>(ng) * static_cast<float>(gsize[gi]) *
                      static_cast<float>(ni));
    } else {
      const unsigned long long nt = scal[1];
      if (nt > 0) c = __frcp_rn(static_cast<float>(nt));
    }
    const float A = adv[i];
    // a lane sums its own tokens and the warp its lanes in fp32 (fixed
    // butterfly); the sums over sequences are fp64
    float s_l = 0.f, s_rho = 0.f, s_kl = 0.f;
    int n_clip = 0;
    // a lane's tokens b + lane, b + lane + 32, ... in order, four loads in flight
    for (int t0 = b + lane; t0 < e; t0 += 128) {
      uint8_t mk[4];
      float lpv[4], olv[4], rfv[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int t = t0 + 32 * u;
        mk[u] = t < e ? lm[t] : 0;
        lpv[u] = mk[u] ? logp[t] : 0.f;
        olv[u] = mk[u] ? old_logp[t] : 0.f;
        rfv[u] = mk[u] && use_kl ? ref_logp[t] : 0.f;
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int t = t0 + 32 * u;
        if (t >= e) break;
        if (!mk[u]) {
          g[t] = 0.f;
          continue;
        }
        const float lp = lpv[u];
        const float rho = expf(lp - olv[u]);
        const float clipped = fminf(fmaxf(rho, lo), hi);
        const float surr = fminf(rho * A, clipped * A);
        const bool binds = (A > 0.f && rho > hi) || (A < 0.f && rho < lo);
        float kl = 0.f, dkl = 0.f;
        if (use_kl) {
          const float delta = rfv[u] - lp;
          const float em1 = expm1f(delta);
          kl = em1 - delta;  // exp(delta) - delta - 1
          dkl = -em1;        // 1 - exp(delta)
        }
        const float ell = -(surr - kl_beta * kl);
        g[t] = c * ((binds ? 0.f : -A * rho) + (use_kl ? kl_beta * dkl : 0.f));
        s_l += ell;
        s_rho += rho;
        s_kl += kl;
        n_clip += binds ? 1 : 0;
      }
    }
    s_l = warp_sum_f(s_l);
    s_rho = warp_sum_f(s_rho);
    s_kl = warp_sum_f(s_kl);
    n_clip = __reduce_add_sync(0xffffffffu, n_clip);
    if (lane == 0) {
      part[3 * i + 0] = static_cast<double>(s_l) * static_cast<double>(c);
      part[3 * i + 1] = s_rho;
      part[3 * i + 2] = s_kl;
      part_clip[i] = n_clip;
    }
  }
}

// (d) fixed-order sum over sequences in two stages: block k sums the
// sequences of its contiguous chunk (thread-strided, then a fixed tree), and
// one block sums the kLossFinalBlocks block results.  The split depends only
// on n_seq, so the loss is the same bits on any device.
constexpr int kLossFinalBlocks = 64;

__global__ void loss_final_partial_kernel(const double* part, const int* part_clip, int n_seq,
                                          int chunk, double* bpart) {
  __shared__ double sh[kLossThreads];
  const int i0 = blockIdx.x * chunk, i1 = min(n_seq, i0 + chunk);
  double l = 0, r = 0, k = 0, c = 0;
  for (int i = i0 + threadIdx.x; i < i1; i += kLossThreads) {
    l += part[3 * i];
    r += part[3 * i + 1];
    k += part[3 * i + 2];
    c += part_clip[i];
  }
  l = block_sum_d(l, sh);
  r = block_sum_d(r, sh);
  k = block_sum_d(k, sh);
  c = block_sum_d(c, sh);
  if (threadIdx.x == 0) {
    bpart[4 * blockIdx.x + 0] = l;
    bpart[4 * blockIdx.x + 1] = r;
    bpart[4 * blockIdx.x + 2] = k;
    bpart[4 * blockIdx.x + 3] = c;
  }
}

__global__ void loss_final_kernel(const double* bpart, int nb, const unsigned long long* scal,
                                  float* loss, float* stats) {
  __shared__ double sh[kLossThreads];
  double l = 0, r = 0, k = 0, c = 0;
  for (int j = threadIdx.x; j < nb; j += kLossThreads) {
    l += bpart[4 * j];
    r += bpart[4 * j + 1];
    k += bpart[4 * j + 2];
    c += bpart[4 * j + 3];
  }
  l = block_sum_d(l, sh);
  r = block_sum_d(r, sh);
  k = block_sum_d(k, sh);
  c = block_sum_d(c, sh);
  if (threadIdx.x == 0) {
    *loss = static_cast<float>(l);
    if (stats) {
      const double n = static_cast<double>(scal[1]);
      stats[0] = n > 0 ? static_cast<float>(c / n) : 0.f;
      stats[1] = n > 0 ? static_cast<float>(r / n) : 0.f;
      stats[2] = n > 0 ? static_cast<float>(k / n) : 0.f;
      stats[3] = static_cast<float>(n);
    }
  }
}

size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }



std::atomic<long long> g_launches{0};

}  // namespace

// SM count of the current device, cached per ordinal (1 if the query fails:
// grids stay valid, only smaller).
int sm_count() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 1;
  static int cache[64] = {0};
  if (cache[dev] == 0) {
    int n = 0;
    cache[dev] = cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess && n > 0
                     ? n
                     : 1;
  }
  return cache[dev];
}

void note_launches(int n) { g_launches.fetch_add(n, std::memory_order_relaxed); }
long long launches() { return g_launches.load(std::memory_order_relaxed); }

int compact_blocks(long long T) { return static_cast<int>((T + kCompactTile - 1) / kCompactTile); }

cudaError_t launch_compact(int kind, const uint8_t* mask, const int* tgt, const float* g,
                           long long T, int* scratch, int* idx, int* count, cudaStream_t s) {
  const int nb = compact_blocks(T);
  int* counts = scratch;
  int* offsets = scratch + nb;
  compact_count_kernel<<<nb, kCompactThreads, 0, s>>>(kind, mask, tgt, g, T, counts);
  compact_scan_kernel<<<1, kCompactThreads, 0, s>>>(counts, nb, offsets, count);
  compact_write_kernel<<<nb, kCompactThreads, 0, s>>>(kind, mask, tgt, g, T, offsets, idx);
  note_launches(3);
  return cudaGetLastError();
}

cudaError_t launch_gather(const __nv_bfloat16* H, int d, const int* idx, const int* count,
                          int rows_cap, __nv_bfloat16* Hc, const int* tgt, int* tgt_c,
                          long long tgt_off, long long tgt_lim, const float* a, float* a_c,
                          const float* b, float* b_c, cudaStream_t s) {
  const int row_vecs = d / 8;  // 16-byte pieces per row
  const int sms = sm_count();
  const int blocks = max(1, min((rows_cap + 7) / 8, sms * 8));
  gather_kernel<<<blocks, 256, 0, s>>>(reinterpret_cast<const uint4*>(H), row_vecs, idx, count,
                                       rows_cap, reinterpret_cast<uint4*>(Hc), tgt, tgt_c,
                                       tgt_off, tgt_lim, a, a_c, b, b_c);
  note_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_lse_combine(const float* partials, int nsplit, const float* ztgt,
                               const int* idx, const int* count, int rows_cap, float* logp,
                               float* entropy, float* lse, const int* tgt_c, float4* rec,
                               cudaStream_t s) {
  const int blocks = (rows_cap + kCombineRows - 1) / kCombineRows;
  lse_combine_kernel<<<blocks, 256, 0, s>>>(partials, nsplit, ztgt, idx, count, logp, entropy, lse,
                                            tgt_c, rec);
  note_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_form_g(__nv_bfloat16* E, long long ldE, int V, int rows_cap,
                          const float* partials, int nsplit, const int* idx, const int* count,
                          const int* tgt_c, const float* lse, const float* g, float inv_temp,
                          cudaStream_t s) {
  const long long work = static_cast<long long>(rows_cap) * (V / 8);
  const int blocks = static_cast<int>(max(1ll, min((work + 255) / 256, 16ll * sm_count())));
  form_g_kernel<<<blocks, 256, 0, s>>>(E, ldE, V, partials, nsplit, idx, count, tgt_c, lse, g,
                                       inv_temp);
  note_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_merge_slices(const float4* rec, int n_slices, long long T, float* logp,
                                float* entropy, float* lse, cudaStream_t s) {
  const long long blocks = (T + 255) / 256;
  merge_slices_kernel<<<static_cast<unsigned>(blocks), 256, 0, s>>>(rec, n_slices, T, logp,
                                                                    entropy, lse);
  note_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_token_select(const int* cu_seqlens, const uint8_t* mask, const int* tgt,
                                int n_seq, int window, uint8_t* loss_mask, int* n_tok,
                                cudaStream_t s) {
  const int warps = 8;
  token_select_kernel<<<(n_seq + warps - 1) / warps, warps * 32, 0, s>>>(
      cu_seqlens, mask, tgt, n_seq, window, loss_mask, n_tok);
  note_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_group_advantages(const float* rewards, const int* group_id, int n_seq,
                                    int n_groups, int std_mode, float eps, float* adv,
                                    cudaStream_t s) {
  const int warps = 4;
  group_adv_kernel<<<(n_groups + warps - 1) / warps, warps * 32, 0, s>>>(
      rewards, group_id, n_seq, n_groups, std_mode, eps, adv);
  note_launches(1);
  return cudaGetLastError();
}

size_t adv_ws_bytes(int n_groups) { return align256(sizeof(int) * (3 * static_cast<size_t>(n_groups) + 1)); }

cudaError_t launch_group_advantages_runs(const float* rewards, const int* group_id, int n_seq,
                                         int n_groups, int std_mode, float eps, float* adv,
                                         void* ws, cudaStream_t s) {
  int* runs = static_cast<int*>(ws);
  int* start = runs + n_groups;
  int* end = start + n_groups;
  int* split = end + n_groups;
  cudaError_t e = cudaMemsetAsync(runs, 0, sizeof(int) * n_groups, s);
  if (e == cudaSuccess) e = cudaMemsetAsync(split, 0, sizeof(int), s);
  if (e != cudaSuccess) return e;
  const int sms = sm_count();
  adv_runs_kernel<<<max(1, min((n_seq + 1023) / 1024, sms * 8)), 256, 0, s>>>(
      group_id, n_seq, n_groups, runs, start, end);
  adv_split_kernel<<<max(1, min((n_groups + 255) / 256, sms * 4)), 256, 0, s>>>(runs, n_groups,
                                                                               split);
  // enough warps for the per-group scan of the fallback, one thread per group otherwise
  const int blocks2 = max(1, min((n_groups + 7) / 8, sms * 16));
  group_adv_runs_kernel<<<blocks2, 256, 0, s>>>(rewards, group_id, n_seq, n_groups, std_mode, eps,
                                                runs, start, end, split, adv);
  note_launches(3);
  return cudaGetLastError();
}

cudaError_t launch_reward_compose(const uint8_t* compiled, const float* pass_rate,
                                  const float* speedup, const float* cv, const float* r_struct,
                                  int n, const RewardParams& q, float* out, cudaStream_t s) {
  const int sms = sm_count();
  auto al = [](const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; };
  const bool vec = al(compiled, 4) && al(pass_rate, 16) && al(speedup, 16) && al(cv, 16) &&
                   al(out, 16) && (r_struct == nullptr || al(r_struct, 16));
  const int n4 = vec ? n / 4 : 0;
  if (n4 > 0) {
    const int blocks = max(1, min((n4 + 255) / 256, sms * 16));
    reward_kernel_x4<<<blocks, 256, 0, s>>>(
        reinterpret_cast<const uchar4*>(compiled), reinterpret_cast<const float4*>(pass_rate),
        reinterpret_cast<const float4*>(speedup), reinterpret_cast<const float4*>(cv),
        reinterpret_cast<const float4*>(r_struct), n4, q, reinterpret_cast<float4*>(out));
    note_launches(1);
  }
  const int done = 4 * n4;
  if (done < n) {
    const int rest = n - done;
    const int blocks = max(1, min((rest + 255) / 256, sms * 8));
    reward_kernel<<<blocks, 256, 0, s>>>(compiled + done, pass_rate + done, speedup + done,
                                         cv + done, r_struct ? r_struct + done : nullptr, rest, q,
                                         out + done);
    note_launches(1);
  }
  return cudaGetLastError();
}

cudaError_t launch_scale(float* x, long long n, float alpha, const float* alpha_dev, cudaStream_t s) {
  const int sms = sm_count();
  const long long want = (n + 255) / 256;
  const int blocks = static_cast<int>(want < sms * 8 ? (want < 1 ? 1 : want) : sms * 8);
  scale_kernel<<<blocks, 256, 0, s>>>(x, n, alpha, alpha_dev);
  note_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_validate(const int* tgt, long long T, long long V, const int* cu, int n_seq,
                            const int* gid, int n_groups, const float* rewards, const float* old_logp,
                            const float* ref_logp, const uint8_t* mask, int* counts, cudaStream_t s) {
  cudaError_t e = cudaMemsetAsync(counts, 0, 6 * sizeof(int), s);
  if (e != cudaSuccess) return e;
  const int sms = sm_count();
  const long long n = T > n_seq ? T : n_seq;
  const long long want = (n + 255) / 256;
  const int blocks = static_cast<int>(want < sms * 4 ? (want < 1 ? 1 : want) : sms * 4);
  validate_kernel<<<blocks, 256, 0, s>>>(tgt, T, V, cu, n_seq, gid, n_groups, rewards, old_logp,
                                         ref_logp, mask, counts);
  note_launches(1);
  return cudaGetLastError();
}

size_t loss_ws_bytes(int n_seq, int n_groups) {
  return align256(sizeof(int) * n_groups) + align256(sizeof(int) * n_seq) +
         align256(2 * sizeof(long long)) + align256(3 * sizeof(double) * n_seq) +
         align256(sizeof(int) * n_seq) + align256(4 * sizeof(double) * kLossFinalBlocks);
}

LossWs carve_loss_ws(void* ws, int n_seq, int n_groups) {
  char* p = static_cast<char*>(ws);
  LossWs w;
  w.gsize = reinterpret_cast<int*>(p);
  p += align256(sizeof(int) * n_groups);
  w.n_tok = reinterpret_cast<int*>(p);
  p += align256(sizeof(int) * n_seq);
  w.scal = reinterpret_cast<unsigned long long*>(p);
  p += align256(2 * sizeof(long long));
  w.part = reinterpret_cast<double*>(p);
  p += align256(3 * sizeof(double) * n_seq);
  w.part_clip = reinterpret_cast<int*>(p);
  p += align256(sizeof(int) * n_seq);
  w.bpart = reinterpret_cast<double*>(p);
  return w;
}

cudaError_t launch_policy_loss(const float* logp, const float* old_logp, const float* ref_logp,
                               const float* adv, const int* cu_seqlens, const int* group_id,
                               int n_seq, int n_groups, const uint8_t* loss_mask, long long T,
                               float clip_eps, float kl_beta, int agg, float* loss, float* g,
                               float* stats, const LossWs& w, cudaStream_t s) {
  (void)T;
  cudaError_t e = cudaMemsetAsync(w.gsize, 0, sizeof(int) * n_groups, s);
  if (e == cudaSuccess) e = cudaMemsetAsync(w.scal, 0, 2 * sizeof(unsigned long long), s);
  if (e != cudaSuccess) return e;
  const int sms = sm_count();
  const int per_block = kLossThreads / 32;  // sequences in flight per block
  const int seq_blocks = max(1, min((n_seq + per_block - 1) / per_block, sms * 8));
  loss_count_kernel<<<seq_blocks, kLossThreads, 0, s>>>(cu_seqlens, group_id, loss_mask, n_seq,
                                                        n_groups, w.n_tok, w.gsize);
  const int nmax = n_seq > n_groups ? n_seq : n_groups;
  loss_scalars_kernel<<<max(1, min((nmax + kLossThreads - 1) / kLossThreads, sms * 4)), kLossThreads,
                        0, s>>>(w.gsize, n_groups, w.n_tok, n_seq, w.scal);
  loss_token_kernel<<<seq_blocks, kLossThreads, 0, s>>>(logp, old_logp, ref_logp, adv, cu_seqlens,
                                                        group_id, n_seq, n_groups, loss_mask,
                                                        clip_eps, kl_beta, agg, w.n_tok, w.gsize,
                                                        w.scal, g, w.part, w.part_clip);
  const int chunk = (n_seq + kLossFinalBlocks - 1) / kLossFinalBlocks;
  const int nb = (n_seq + chunk - 1) / chunk;
  loss_final_partial_kernel<<<nb, kLossThreads, 0, s>>>(w.part, w.part_clip, n_seq, chunk,
                                                        w.bpart);
  loss_final_kernel<<<1, kLossThreads, 0, s>>>(w.bpart, nb, w.scal, loss, stats);
  note_launches(5);
  return cudaGetLastError();
}

}  // namespace spo
