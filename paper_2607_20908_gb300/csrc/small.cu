// small.cu -- the bandwidth- and latency-bound steps of the path: loss-token
// selection, row compaction and gather, the split-vocabulary logsumexp
// combine, group-normalised advantages and the policy-loss forward.
#include <math.h>

#include <atomic>

#include "internal.h"
#include "tc.cuh"

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
__device__ __forceinline__ int group_adv_warp(const float* rewards, const int* gid, int g, int b,
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
  return n;  // the group's member count (the same in every lane)
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
// end of its run (meaningful when it has one); raises *split when a group
// has a second run (its members are not contiguous).  Runs only when the
// sorted pass found the ids out of order.
__global__ void adv_runs_kernel(const int* gid, int n_seq, int n_groups, int* runs, int* start,
                                int* end, int* split, const int* unsorted) {
  if (!*unsorted) return;
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
        if (atomicAdd(&runs[g], 1) > 0) *split = 1;
        start[g] = i;
      }
      if (i == n_seq - 1 || gn[u] != g) end[g] = i + 1;
    }
  }
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

// The same fold for a group of n <= N members held in registers: each member
// is read once, and the three passes run over the registers (predicated on
// u < n, in ascending order: the same operations as group_adv_thread).
template <int N, class At>
__device__ __forceinline__ void group_adv_regs(float* s, int b, int n, int std_mode, float eps,
                                               At at) {
  float r[N];
#pragma unroll
  for (int u = 0; u < N; ++u) r[u] = u < n ? s[at(b + u)] : 0.f;
  float acc = 0.f, lo = INFINITY, hi = -INFINITY;
#pragma unroll
  for (int u = 0; u < N; ++u) {
    if (u < n) {
      acc = __fadd_rn(acc, r[u]);
      lo = fminf(lo, r[u]);
      hi = fmaxf(hi, r[u]);
    }
  }
  const bool zero = n <= 1 || lo == hi;
  float mu = 0.f, den = 1.f;
  if (!zero) {
    mu = __fdiv_rn(acc, static_cast<float>(n));
    float ss = 0.f;
#pragma unroll
    for (int u = 0; u < N; ++u) {
      if (u < n) {
        const float dv = __fsub_rn(r[u], mu);
        ss = __fadd_rn(ss, __fmul_rn(dv, dv));
      }
    }
    const float var = __fdiv_rn(ss, static_cast<float>(std_mode == 0 ? n - 1 : n));
    den = __fadd_rn(__fsqrt_rn(var), eps);
  }
#pragma unroll
  for (int u = 0; u < N; ++u)
    if (u < n) s[at(b + u)] = zero ? 0.f : __fdiv_rn(__fsub_rn(r[u], mu), den);
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
    const int* runs, const int* start, const int* end, const int* split, const int* unsorted,
    float* adv) {
  __shared__ float st[kAdvStage + kAdvStage / 32];
  if (!*unsorted) return;
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

// End of the run of group g that starts at b, for non-decreasing ids: the
// first index past b whose id differs (or n).  Probes b + 1, b + 2, b + 4, ...
// and then bisects, so a run of length L costs O(log L) loads.  On ids that
// are not sorted it still returns an index in (b, n]; the caller's result is
// then replaced by the run path.
__device__ int adv_run_end(const int* gid, int b, int n, int g) {
  int lo = b + 1, hi = n;  // gid[lo - 1] == g; the end lies in [lo, hi]
  for (int step = 1;; step <<= 1) {
    const long long p = static_cast<long long>(b) + step;
    if (p < n && gid[p] == g) {
      lo = static_cast<int>(p) + 1;
    } else {
      hi = static_cast<int>(p < n ? p : n);
      break;
    }
  }
  while (lo < hi) {
    const int mid = lo + (hi - lo) / 2;
    if (gid[mid] == g) lo = mid + 1;
    else hi = mid;
  }
  return lo;
}

// Sorted pass of the run path: one block per chunk of kAdvChunk consecutive
// sequences.  The block stages the chunk's rewards (padded, as in the run
// kernel) and ids, plus the id before it and a halo of kAdvHalo sequences
// after it, in shared memory with coalesced loads, and checks that every id
// of the chunk is in [0, n_groups) and none is below its predecessor; if one
// is, it raises *unsorted and the run path recomputes every advantage.
// Otherwise each group is one run: the groups that start in the chunk are
// found with ballots and a block scan, each is folded by one thread in
// ascending index (group_adv_thread: the same bits), and the advantages go
// back with coalesced stores.  The chunk's last group may run on past its
// end: if it ends inside the halo it is folded there too, else it is folded
// from memory.  Sequences before the chunk's first start belong to an
// earlier block.  The block also clears its share of the run counters for
// the run path.
constexpr int kAdvChunk = 4096;
constexpr int kAdvHalo = 256;  // one sequence per thread
constexpr int kAdvStaged = kAdvChunk + kAdvHalo;

__global__ void __launch_bounds__(256, 6) adv_sorted_kernel(const float* rewards, const int* gid,
                                                         int n_seq, int n_groups, int std_mode,
                                                         float eps, float* adv, int* runs,
                                                         int* unsorted) {
  __shared__ float st[kAdvStaged + kAdvStaged / 32];
  __shared__ int sg[kAdvStaged + 1];  // ids of [c0 - 1, c1 + halo); then the list of group starts
  __shared__ unsigned starts[kAdvChunk / 32];
  __shared__ int tail_end;
  const int tid = threadIdx.x;
  for (int g = blockIdx.x * blockDim.x + tid; g < n_groups; g += gridDim.x * blockDim.x) runs[g] = 0;
  const int c0 = blockIdx.x * kAdvChunk;
  const int len = min(kAdvChunk, n_seq - c0);
  const int staged = min(kAdvStaged, n_seq - c0);  // chunk + halo
  const AtPadded at;
#pragma unroll 8
  for (int k = tid; k < staged; k += 256) {
    sg[k + 1] = gid[c0 + k];
    st[at(k)] = rewards[c0 + k];
  }
  if (tid == 0) {
    sg[0] = c0 > 0 ? gid[c0 - 1] : -1;
    tail_end = INT_MAX;
  }
  __syncthreads();
  // bit k of the chunk's start mask: a group starts at c0 + k
  bool bad = false;
#pragma unroll
  for (int j = 0; j < kAdvChunk / 256; ++j) {
    const int k = j * 256 + tid;
    const bool in = k < len;
    const int g = in ? sg[k + 1] : 0, gp = in ? sg[k] : 0;
    bad |= in && (g < 0 || g >= n_groups || (c0 + k > 0 && g < gp));
    const unsigned m = __ballot_sync(0xffffffffu, in && g != gp);
    if ((tid & 31) == 0) starts[j * 8 + (tid >> 5)] = m;
  }
  if (__syncthreads_or(bad)) {
    if (tid == 0) atomicOr(unsorted, 1);
    return;
  }
  // the last group runs on past the chunk when the next id is the same; its
  // end is the first halo position with another id
  const bool straddle = len < staged && sg[len] == sg[len + 1];
  const int g_tail = sg[len];
  if (straddle && len + tid < staged && sg[len + tid + 1] != g_tail) atomicMin(&tail_end, len + tid);
  __syncthreads();
  const unsigned word = tid < kAdvChunk / 32 ? starts[tid] : 0u;
  int n_starts = 0;
  int o = block_exclusive_scan(__popc(word), &n_starts);  // ends with a barrier: sg is free
  // inside the halo, at the end of the data, or (-1) beyond the halo
  const int e_tail = tail_end != INT_MAX ? tail_end : (c0 + staged == n_seq ? staged : -1);
  int* list = sg;
  for (unsigned w = word; w; w &= w - 1u) list[o++] = tid * 32 + __ffs(w) - 1;
  __syncthreads();
  for (int q0 = 0; q0 < n_starts; q0 += 256) {
    // thread q0 + tid folds group q in shared memory, in registers when the
    // largest group of its warp has at most 16 members; a last group that runs
    // past the halo is folded from memory
    const int q = q0 + tid;
    const bool live = q < n_starts;
    const int b = live ? list[q] : 0;
    const int e = !live ? 0 : q + 1 < n_starts ? list[q + 1] : !straddle ? len : e_tail;
    const bool from_memory = live && e < 0;
    const int n = live && !from_memory ? e - b : 0;
    const int n_max = __reduce_max_sync(0xffffffffu, n);
    if (n_max <= 4) group_adv_regs<4>(st, b, n, std_mode, eps, at);
    else if (n_max <= 8) group_adv_regs<8>(st, b, n, std_mode, eps, at);
    else if (n_max <= 16) group_adv_regs<16>(st, b, n, std_mode, eps, at);
    else if (n > 0) group_adv_thread(st, b, e, std_mode, eps, st, at);
    if (from_memory) {
      const int end = adv_run_end(gid, c0 + b, n_seq, g_tail);
      group_adv_thread(rewards, c0 + b, end, std_mode, eps, adv, AtIdentity());
    }
  }
  __syncthreads();
  // the groups that start in this chunk, the last one into the halo when it ends there
  const int wb_lo = n_starts > 0 ? list[0] : len;
  const int wb_hi = !straddle || n_starts == 0 ? len : e_tail >= 0 ? e_tail : list[n_starts - 1];
  for (int k = wb_lo + tid; k < wb_hi; k += 256) adv[c0 + k] = st[at(k)];
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

// x *= num / den (counts in fp64; 0 when den is 0): a data-parallel rank's
// weight in the global average, taken from all-reduced counts on the device.
__global__ void scale_ratio_kernel(float* x, long long n, const double* num, const double* den) {
  const double dd = *den;
  const float a = dd != 0.0 ? static_cast<float>(*num / dd) : 0.f;
  for (long long i = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<long long>(gridDim.x) * blockDim.x)
    x[i] *= a;
}

__global__ void scale_kernel(float* x, long long n, float alpha, const float* alpha_dev) {
  const float a = alpha_dev ? *alpha_dev : alpha;
  for (long long i = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<long long>(gridDim.x) * blockDim.x)
    x[i] *= a;
}

// Rows of dH that the backward skips (g == 0, the complement of its row
// compaction) are zeroed here, one warp per token row with 16-byte stores; the
// dH GEMM writes every other row.
__global__ void zero_skipped_rows_kernel(const float* g, long long T, int row_bytes, uint8_t* out) {
  const int lane = threadIdx.x & 31;
  const long long nw = (static_cast<long long>(gridDim.x) * blockDim.x) >> 5;
  for (long long t = (blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x) >> 5; t < T;
       t += nw) {
    if (g[t] != 0.f) continue;  // the same test as the compaction; uniform across the warp
    uint4* row = reinterpret_cast<uint4*>(out + t * row_bytes);
    for (int k = lane; k < row_bytes / 16; k += 32) row[k] = make_uint4(0u, 0u, 0u, 0u);
  }
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

// Global warp index and warp count of the grid (the loss kernels' sequence
// groups are derived from them; the grid strides over sequences).
__device__ __forceinline__ int warp_seq0() { return (blockIdx.x * blockDim.x + threadIdx.x) >> 5; }
__device__ __forceinline__ int warp_seq_stride() { return (gridDim.x * blockDim.x) >> 5; }

__device__ __forceinline__ long long warp_sum_ll(long long v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// (a) sequences per group and the number of non-empty groups; for the token
// mean also the number of loss tokens of [cu[0], cu[n_seq]) (integers; the
// counters were cleared on the stream).  Each phase of the launch strides over
// the whole grid.
__device__ __forceinline__ int nonzero_bytes(unsigned w) {
  // high bit of each byte set iff the byte is non-zero (no carry crosses bytes)
  return __popc((((w & 0x7f7f7f7fu) + 0x7f7f7f7fu) | w) & 0x80808080u);
}

__device__ __forceinline__ long long grid_tid() {
  return static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
}
__device__ __forceinline__ long long grid_threads() {
  return static_cast<long long>(gridDim.x) * blockDim.x;
}

// Loss tokens of [cu[0], cu[n_seq]) counted by this thread: bytes up to the
// first 16-byte-aligned address, then 16 at a time, then the tail.
__device__ __forceinline__ long long count_loss_tokens(const int* cu, int n_seq, const uint8_t* lm) {
  const long long tid = grid_tid(), stride = grid_threads();
  long long nt = 0;
  const long long lo = cu[0], hi = cu[n_seq];
  const long long lead = static_cast<long long>((16u - (reinterpret_cast<uintptr_t>(lm + lo) & 15u)) & 15u);
  const long long a = min(hi, lo + lead);
  const long long z = a + (hi - a) / 16 * 16;
  for (long long t = lo + tid; t < a; t += stride) nt += lm[t] != 0;
  const uint4* v = reinterpret_cast<const uint4*>(lm + a);
  for (long long k = tid; k < (z - a) / 16; k += stride) {
    const uint4 q = __ldcs(v + k);
    nt += nonzero_bytes(q.x) + nonzero_bytes(q.y) + nonzero_bytes(q.z) + nonzero_bytes(q.w);
  }
  for (long long t = z + tid; t < hi; t += stride) nt += lm[t] != 0;
  return nt;
}

// One update of each counter per block (same-address atomics serialise).
__device__ __forceinline__ void add_block_counts(long long first, long long nt,
                                                 unsigned long long* scal) {
  __shared__ long long sf[kLossThreads / 32], st[kLossThreads / 32];
  first = warp_sum_ll(first);
  nt = warp_sum_ll(nt);
  if ((threadIdx.x & 31) == 0) {
    sf[threadIdx.x >> 5] = first;
    st[threadIdx.x >> 5] = nt;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    long long f = 0, n = 0;
    for (int w = 0; w < kLossThreads / 32; ++w) {
      f += sf[w];
      n += st[w];
    }
    if (f) atomicAdd(&scal[0], static_cast<unsigned long long>(f));
    if (n) atomicAdd(&scal[1], static_cast<unsigned long long>(n));
  }
}

__device__ __forceinline__ void loss_group_counts(const int* gid, int n_seq, int n_groups,
                                                  const int* cu, const uint8_t* lm, int agg,
                                                  int* gsize, unsigned long long* scal) {
  const long long tid = grid_tid(), stride = grid_threads();
  long long first = 0;
  for (long long i = tid; i < n_seq; i += stride) {
    const int g = gid[i];
    if (g >= 0 && g < n_groups && atomicAdd(&gsize[g], 1) == 0) ++first;
  }
  add_block_counts(first, agg == 1 ? count_loss_tokens(cu, n_seq, lm) : 0, scal);
}

// The same counts together with the group advantages (a4), for a step's few
// hundred sequences: warp w of the grid folds groups w, w + warps, ... with
// group_adv_warp (the per-group scan of spo_group_advantages: the same bits)
// and records each group's size, so the sizes need no atomics.
__device__ __forceinline__ void adv_and_group_counts(const float* rewards, const int* gid,
                                                     int n_seq, int n_groups, int std_mode,
                                                     float eps, float* adv, const int* cu,
                                                     const uint8_t* lm, int agg, int* gsize,
                                                     unsigned long long* scal) {
  const int lane = threadIdx.x & 31;
  const int warps = static_cast<int>(grid_threads() >> 5);
  long long first = 0;
  for (int g = static_cast<int>(grid_tid() >> 5); g < n_groups; g += warps) {
    const int n = group_adv_warp(rewards, gid, g, 0, n_seq, true, std_mode, eps, adv, lane);
    if (lane == 0) {
      gsize[g] = n;
      first += n > 0;
    }
  }
  add_block_counts(first, agg == 1 ? count_loss_tokens(cu, n_seq, lm) : 0, scal);
}

// (b) per-token surrogate, KL, dL/dlogp; per-sequence sums.  A group of LPS
// lanes takes one sequence (LPS = 16 when sequences average at most 128
// tokens, so a warp holds two at once; else the whole warp) in passes of
// 8 tokens a lane: the group counts the sequence's loss tokens (n_i of c_t)
// while the first pass's inputs stay in registers (a sequence of up to 8 LPS
// tokens is read once), then lane l of the group sums its own tokens
// b + l, b + l + LPS, ... in order in fp32 and the group's lanes are
// combined by a fixed xor butterfly.  The next sequence's bounds, group and
// advantage are loaded one sequence ahead.
//
// kl = e^delta - delta - 1 is taken from the Taylor series of e^delta for
// |delta| <= 1/2: kl = delta^2 (1/2! + delta/3! + ... + delta^7/9!) (the
// first omitted term is below 3e-9 of the sum), which also avoids the
// cancellation of e^delta - 1 - delta near 0; beyond, e^delta - 1 - delta
// directly.  e^delta - 1 = delta + kl in both cases.
__device__ __forceinline__ float kl_k3(float delta, float* em1) {
  float kl;
  if (fabsf(delta) <= 0.5f) {
    float p = 1.f / 362880.f;
    p = fmaf(p, delta, 1.f / 40320.f);
    p = fmaf(p, delta, 1.f / 5040.f);
    p = fmaf(p, delta, 1.f / 720.f);
    p = fmaf(p, delta, 1.f / 120.f);
    p = fmaf(p, delta, 1.f / 24.f);
    p = fmaf(p, delta, 1.f / 6.f);
    p = fmaf(p, delta, 0.5f);
    kl = delta * delta * p;
    *em1 = delta + kl;
  } else {
    *em1 = expf(delta) - 1.f;
    kl = *em1 - delta;
  }
  return kl;
}

struct LossTok {
  float lo, hi, A, c, beta;
  bool use_kl;
  float s_l = 0.f, s_rho = 0.f, s_kl = 0.f;
  int n_clip = 0;
  __device__ __forceinline__ float token(float lp, float ol, float rf) {
    const float rho = expf(lp - ol);
    const float clipped = fminf(fmaxf(rho, lo), hi);
    const float surr = fminf(rho * A, clipped * A);
    const bool binds = (A > 0.f && rho > hi) || (A < 0.f && rho < lo);
    float kl = 0.f, dkl = 0.f;
    if (use_kl) {
      float em1;
      kl = kl_k3(rf - lp, &em1);
      dkl = -em1;  // d kl / d logp = 1 - e^delta
    }
    s_l += -(surr - beta * kl);
    s_rho += rho;
    s_kl += kl;
    n_clip += binds ? 1 : 0;
    return c * ((binds ? 0.f : -A * rho) + (use_kl ? beta * dkl : 0.f));
  }
};

// Fixed xor butterfly over the LPS lanes of a group (mask m): every lane of
// the group ends with the same bits.
template <int LPS>
__device__ __forceinline__ float group_sum_f(float v, unsigned m) {
#pragma unroll
  for (int o = LPS / 2; o > 0; o >>= 1) v = __fadd_rn(v, __shfl_xor_sync(m, v, o));
  return v;
}

// ld(p): a load of a count or advantage; with IN_LAUNCH (phases of one
// launch) they were written by other blocks earlier in the same launch, so the
// load goes to L2, past this SM's L1.
template <int LPS, bool IN_LAUNCH>
__device__ __forceinline__ void loss_token_pass(
    const float* logp, const float* old_logp, const float* ref_logp, const float* adv,
    const int* cu, const int* gid, int n_seq, int n_groups, const uint8_t* lm, float clip_eps,
    float kl_beta, int agg, const int* gsize, const unsigned long long* scal, const float* cscale,
    float* g, float2* part_l, float2* part_rk, int* part_clip, int* n_tok) {
  constexpr int kTpl = 8;            // tokens a lane has in flight in one pass
  constexpr int kStep = kTpl * LPS;  // tokens of one pass of the group
  const int lane = threadIdx.x & 31;
  const int sl = lane % LPS;
  const unsigned gm = LPS == 32 ? 0xffffffffu : ((1u << LPS) - 1u) << (lane - sl);
  const bool use_kl = ref_logp != nullptr && kl_beta != 0.f;
  auto ld = [](const auto* p) { return IN_LAUNCH ? __ldcg(p) : *p; };
  const unsigned long long n_nonempty = ld(scal), n_loss = ld(scal + 1);
  const float ng = static_cast<float>(n_nonempty);
  const float c_tok = n_loss > 0 ? __frcp_rn(static_cast<float>(n_loss)) : 0.f;
  const int stride = warp_seq_stride() * (32 / LPS);
  int i = warp_seq0() * (32 / LPS) + lane / LPS;
  int b = 0, e = 0, gi = -1;
  float A = 0.f;
  if (i < n_seq) {
    b = cu[i];
    e = cu[i + 1];
    gi = gid[i];
    A = ld(adv + i);
  }
  for (; i < n_seq; i += stride) {
    const int in = i + stride;
    int nb = 0, ne = 0, ngi = -1;
    float nA = 0.f;
    if (in < n_seq) {
      nb = cu[in];
      ne = cu[in + 1];
      ngi = gid[in];
      nA = ld(adv + in);
    }
    const int gs = agg == 0 && gi >= 0 && gi < n_groups ? ld(gsize + gi) : 0;
    // the first pass's inputs stay in registers while the mask is counted
    uint8_t mk[kTpl];
    float lpv[kTpl], olv[kTpl], rfv[kTpl];
#pragma unroll
    for (int u = 0; u < kTpl; ++u) {
      const int t = b + sl + LPS * u;
      const bool inside = t < e;
      mk[u] = inside ? lm[t] : 0;
      lpv[u] = inside ? logp[t] : 0.f;
      olv[u] = inside ? old_logp[t] : 0.f;
      rfv[u] = inside && use_kl ? ref_logp[t] : 0.f;
    }
    int cnt = 0;
#pragma unroll
    for (int u = 0; u < kTpl; ++u) cnt += mk[u] != 0;
    for (int t0 = b + kStep + sl; t0 < e; t0 += kStep) {
#pragma unroll
      for (int u = 0; u < kTpl; ++u) cnt += t0 + LPS * u < e && lm[t0 + LPS * u] != 0;
    }
    const int ni = __reduce_add_sync(gm, cnt);
    // c_t of Eq. 3's average; fp32 (GB300's fp64 unit is narrow, and every
    // lane computes it)
    float c = c_tok;
    if (agg == 0)
      c = ni > 0 && ng > 0.f && gs > 0
              ? __frcp_rn(ng * static_cast<float>(gs) * static_cast<float>(ni))
              : 0.f;
    if (cscale) c *= *cscale;  // a data-parallel rank's share of the global average
    LossTok k{1.f - clip_eps, 1.f + clip_eps, A, c, kl_beta, use_kl};
#pragma unroll
    for (int u = 0; u < kTpl; ++u) {
      const int t = b + sl + LPS * u;
      if (t < e) g[t] = mk[u] ? k.token(lpv[u], olv[u], rfv[u]) : 0.f;
    }
    for (int t0 = b + kStep + sl; t0 < e; t0 += kStep) {
#pragma unroll
      for (int u = 0; u < kTpl; ++u) {
        const int t = t0 + LPS * u;
        const bool inside = t < e;
        mk[u] = inside ? lm[t] : 0;
        lpv[u] = inside ? logp[t] : 0.f;
        olv[u] = inside ? old_logp[t] : 0.f;
        rfv[u] = inside && use_kl ? ref_logp[t] : 0.f;
      }
#pragma unroll
      for (int u = 0; u < kTpl; ++u) {
        const int t = t0 + LPS * u;
        if (t < e) g[t] = mk[u] ? k.token(lpv[u], olv[u], rfv[u]) : 0.f;
      }
    }
    const float s_l = group_sum_f<LPS>(k.s_l, gm);
    const float s_rho = group_sum_f<LPS>(k.s_rho, gm);
    const float s_kl = group_sum_f<LPS>(k.s_kl, gm);
    const int n_clip = __reduce_add_sync(gm, k.n_clip);
    if (sl == 0) {
      const float hi = s_l * c;  // c * s_l as an unevaluated pair: hi + lo exactly
      part_l[i] = make_float2(hi, fmaf(s_l, c, -hi));
      part_rk[i] = make_float2(s_rho, s_kl);
      part_clip[i] = n_clip;
      n_tok[i] = ni;
    }
    b = nb;
    e = ne;
    gi = ngi;
    A = nA;
  }
}

// (c) fixed-order sum over sequences in two stages: block k sums the
// sequences of its contiguous chunk (one per thread at the usual sizes; then
// each warp by a fixed butterfly and the block's warps in order), and the
// last block to finish (a ticket taken after its sums are visible) sums the
// block results the same way in block order.  The loss terms are carried as
// unevaluated pairs of floats (hi + lo, about 48 significant bits) and added
// with Knuth's TwoSum, so cancellation between the terms costs no accuracy
// and GB300's narrow fp64 unit is not used; the ratio and KL statistics are
// summed in fp32, the counts as integers.  The chunk size depends only on
// n_seq, so the results are the same bits on any device.
constexpr int kLossFinalMaxBlocks = 1024;

// (a_hi + a_lo) + (b_hi + b_lo) as a normalised pair (TwoSum of the high
// parts, the low parts added to its error term, then a fast renormalisation)
__device__ __forceinline__ float2 pair_add(float2 a, float2 b) {
  const float s = __fadd_rn(a.x, b.x);
  const float v = __fsub_rn(s, a.x);
  float err = __fadd_rn(__fsub_rn(a.x, __fsub_rn(s, v)), __fsub_rn(b.x, v));
  err = __fadd_rn(err, __fadd_rn(a.y, b.y));
  const float hi = __fadd_rn(s, err);
  return make_float2(hi, __fsub_rn(err, __fsub_rn(hi, s)));
}

struct LossSums {
  float2 l;
  float r, k;
  long long c, n;
  __device__ __forceinline__ void zero() {
    l = make_float2(0.f, 0.f);
    r = k = 0.f;
    c = n = 0;
  }
  __device__ __forceinline__ void add(const LossSums& o) {
    l = pair_add(l, o.l);
    r = __fadd_rn(r, o.r);
    k = __fadd_rn(k, o.k);
    c += o.c;
    n += o.n;
  }
};

__device__ __forceinline__ LossSums block_sums(LossSums v, LossSums* sh) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    LossSums w;
    w.l.x = __shfl_xor_sync(0xffffffffu, v.l.x, o);
    w.l.y = __shfl_xor_sync(0xffffffffu, v.l.y, o);
    w.r = __shfl_xor_sync(0xffffffffu, v.r, o);
    w.k = __shfl_xor_sync(0xffffffffu, v.k, o);
    w.c = __shfl_xor_sync(0xffffffffu, v.c, o);
    w.n = __shfl_xor_sync(0xffffffffu, v.n, o);
    v.add(w);
  }
  if ((threadIdx.x & 31) == 0) sh[threadIdx.x >> 5] = v;
  __syncthreads();
  LossSums t = sh[0];
  for (int w = 1; w < kLossThreads / 32; ++w) t.add(sh[w]);
  __syncthreads();
  return t;
}

// Chunk c of the sequences (fixed split: chunk sequences each, depending only
// on n_seq) summed by the block in a fixed order, then the last block to
// finish (a ticket taken after its sums are visible) sums the chunks' results
// in chunk order.  Per-sequence partials written by other blocks earlier in
// the launch are read through L2.
__device__ __forceinline__ void loss_final_phase(const float2* part_l, const float2* part_rk,
                                                 const int* part_clip, const int* n_tok,
                                                 int n_seq, int chunk, int nb, LossSums* bpart,
                                                 unsigned long long* ticket, float* loss,
                                                 float* stats) {
  __shared__ LossSums sh[kLossThreads / 32];
  __shared__ bool last;
  for (int c = blockIdx.x; c < nb; c += gridDim.x) {
    const int i0 = c * chunk, i1 = min(n_seq, i0 + chunk);
    LossSums v;
    v.zero();
    for (int i = i0 + threadIdx.x; i < i1; i += kLossThreads) {
      LossSums q;
      q.l = __ldcg(part_l + i);
      const float2 rk = __ldcg(part_rk + i);
      q.r = rk.x;
      q.k = rk.y;
      q.c = __ldcg(part_clip + i);
      q.n = __ldcg(n_tok + i);
      v.add(q);
    }
    v = block_sums(v, sh);
    if (threadIdx.x == 0) bpart[c] = v;
  }
  if (threadIdx.x == 0) {
    __threadfence();
    last = atomicAdd(ticket, 1ull) == gridDim.x - 1;
  }
  __syncthreads();
  if (!last) return;
  __threadfence();
  LossSums u;
  u.zero();
  for (int j = threadIdx.x; j < nb; j += kLossThreads) {
    const volatile LossSums* q = bpart + j;
    LossSums x;
    x.l.x = q->l.x;
    x.l.y = q->l.y;
    x.r = q->r;
    x.k = q->k;
    x.c = q->c;
    x.n = q->n;
    u.add(x);
  }
  u = block_sums(u, sh);
  if (threadIdx.x == 0) {
    *loss = __fadd_rn(u.l.x, u.l.y);
    if (stats) {
      const double n = static_cast<double>(u.n);
      stats[0] = n > 0 ? static_cast<float>(static_cast<double>(u.c) / n) : 0.f;
      stats[1] = n > 0 ? static_cast<float>(static_cast<double>(u.r) / n) : 0.f;
      stats[2] = n > 0 ? static_cast<float>(static_cast<double>(u.k) / n) : 0.f;
      stats[3] = static_cast<float>(n);
    }
  }
}

// Grid-wide barrier of a cooperative launch (every block resident): each
// block arrives once on *count and waits until `target` arrivals.  The wait
// is bounded: past kWaitTimeoutNs the block records kErrWaitGridBarrier in the
// device error word and the caller returns (its outputs are then undefined,
// and spo_device_error / spo_sync_check report the timeout).
__device__ __forceinline__ bool grid_barrier(unsigned long long* count, unsigned long long target,
                                             int* err) {
  __shared__ int ok_s;
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    atomicAdd(count, 1ull);
    const unsigned long long t0 = globaltimer();
    int ok = 1;
    while (ld_relaxed_gpu_u64(count) < target) {
      if (globaltimer() - t0 > kWaitTimeoutNs) {
        ok = 0;
        if (err) atomicCAS(err, 0, kErrWaitGridBarrier);
        break;
      }
      __nanosleep(32);
    }
    __threadfence();
    ok_s = ok;
  }
  __syncthreads();
  return ok_s != 0;
}

// The loss forward as one cooperative launch: (a) group sizes and counts --
// with the group advantages too when WITH_ADV -- then (b) the token pass,
// then (c) the fixed-order sum, a grid barrier between phases.  The phases
// compute exactly what separate launches of them would.
struct LossLaunch {
  const float* logp;
  const float* old_logp;
  const float* ref_logp;
  const float* adv;      // in, or (WITH_ADV) written by phase (a)
  float* adv_out;
  const float* rewards;  // WITH_ADV
  int std_mode;
  float adv_eps;
  const int* cu;
  const int* gid;
  int n_seq;
  int n_groups;
  const uint8_t* lm;
  float clip_eps;
  float kl_beta;
  int agg;
  const float* cscale;
  float* loss;
  float* g;
  float* stats;
  LossWs w;
  int chunk;
  int nb;
  int* err;
};

template <int LPS, bool WITH_ADV>
__global__ void __launch_bounds__(kLossThreads) loss_fused_kernel(const LossLaunch a) {
  unsigned long long* bar = a.w.scal + 3;
  if (WITH_ADV)
    adv_and_group_counts(a.rewards, a.gid, a.n_seq, a.n_groups, a.std_mode, a.adv_eps, a.adv_out,
                         a.cu, a.lm, a.agg, a.w.gsize, a.w.scal);
  else
    loss_group_counts(a.gid, a.n_seq, a.n_groups, a.cu, a.lm, a.agg, a.w.gsize, a.w.scal);
  if (!grid_barrier(bar, gridDim.x, a.err)) return;
  loss_token_pass<LPS, true>(a.logp, a.old_logp, a.ref_logp, a.adv, a.cu, a.gid, a.n_seq,
                             a.n_groups, a.lm, a.clip_eps, a.kl_beta, a.agg, a.w.gsize, a.w.scal,
                             a.cscale, a.g, a.w.part_l, a.w.part_rk, a.w.part_clip, a.w.n_tok);
  if (!grid_barrier(bar, 2ull * gridDim.x, a.err)) return;
  loss_final_phase(a.w.part_l, a.w.part_rk, a.w.part_clip, a.w.n_tok, a.n_seq, a.chunk, a.nb,
                   static_cast<LossSums*>(a.w.bpart), a.w.scal + 2, a.loss, a.stats);
}

// The same three phases as separate launches, for batches of more sequences
// than a cooperative launch is worth (the phases then fill the device
// independently and nothing waits at a grid barrier).
template <bool WITH_ADV>
__global__ void __launch_bounds__(kLossThreads) loss_counts_kernel(const LossLaunch a) {
  if (WITH_ADV)
    adv_and_group_counts(a.rewards, a.gid, a.n_seq, a.n_groups, a.std_mode, a.adv_eps, a.adv_out,
                         a.cu, a.lm, a.agg, a.w.gsize, a.w.scal);
  else
    loss_group_counts(a.gid, a.n_seq, a.n_groups, a.cu, a.lm, a.agg, a.w.gsize, a.w.scal);
}

template <int LPS>
__global__ void __launch_bounds__(kLossThreads, 4) loss_token_kernel(const LossLaunch a) {
  loss_token_pass<LPS, false>(a.logp, a.old_logp, a.ref_logp, a.adv, a.cu, a.gid, a.n_seq,
                              a.n_groups, a.lm, a.clip_eps, a.kl_beta, a.agg, a.w.gsize, a.w.scal,
                              a.cscale, a.g, a.w.part_l, a.w.part_rk, a.w.part_clip, a.w.n_tok);
}

__global__ void __launch_bounds__(kLossThreads) loss_final_kernel(const LossLaunch a) {
  loss_final_phase(a.w.part_l, a.w.part_rk, a.w.part_clip, a.w.n_tok, a.n_seq, a.chunk, a.nb,
                   static_cast<LossSums*>(a.w.bpart), a.w.scal + 2, a.loss, a.stats);
}

// Sequences up to which the loss forward is one cooperative launch.
constexpr int kLossFusedMaxSeq = 16384;

size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }



std::atomic<long long> g_launches{0};

}  // namespace

// SM count of the current device, cached per ordinal (1 if the query fails:
// grids stay valid, only smaller).
int sm_count() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 1;
  static std::atomic<int> cache[64] = {};  // racing first calls store the same value
  int c = cache[dev].load(std::memory_order_relaxed);
  if (c == 0) {
    int n = 0;
    c = cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess && n > 0 ? n : 1;
    cache[dev].store(c, std::memory_order_relaxed);
  }
  return c;
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

size_t adv_ws_bytes(int n_groups) { return align256(sizeof(int) * (3 * static_cast<size_t>(n_groups) + 2)); }

cudaError_t launch_group_advantages_runs(const float* rewards, const int* group_id, int n_seq,
                                         int n_groups, int std_mode, float eps, float* adv,
                                         void* ws, cudaStream_t s) {
  int* runs = static_cast<int*>(ws);
  int* start = runs + n_groups;
  int* end = start + n_groups;
  int* split = end + n_groups;  // [0]: some group has several runs; [1]: ids out of order
  int* unsorted = split + 1;
  cudaError_t e = cudaMemsetAsync(split, 0, 2 * sizeof(int), s);
  if (e != cudaSuccess) return e;
  const int sms = sm_count();
  adv_sorted_kernel<<<(n_seq + kAdvChunk - 1) / kAdvChunk, 256, 0, s>>>(
      rewards, group_id, n_seq, n_groups, std_mode, eps, adv, runs, unsorted);
  // the run path: each kernel returns at once when the sorted pass succeeded,
  // so its grid is one block per SM (grid-stride loops)
  adv_runs_kernel<<<max(1, min((n_seq + 1023) / 1024, sms)), 256, 0, s>>>(
      group_id, n_seq, n_groups, runs, start, end, split, unsorted);
  const int blocks2 = max(1, min((n_groups + 7) / 8, sms));
  group_adv_runs_kernel<<<blocks2, 256, 0, s>>>(rewards, group_id, n_seq, n_groups, std_mode, eps,
                                                runs, start, end, split, unsorted, adv);
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

cudaError_t launch_scale_ratio(float* x, long long n, const double* num, const double* den,
                               cudaStream_t s) {
  const int sms = sm_count();
  const long long want = (n + 255) / 256;
  const int blocks = static_cast<int>(want < sms * 8 ? (want < 1 ? 1 : want) : sms * 8);
  scale_ratio_kernel<<<blocks, 256, 0, s>>>(x, n, num, den);
  note_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_zero_skipped_rows(const float* g, long long T, int row_bytes, void* out,
                                     cudaStream_t s) {
  const int sms = sm_count();
  const long long want = (T + 7) / 8;  // 8 rows (warps) per block
  const int blocks = static_cast<int>(want < sms * 16ll ? (want < 1 ? 1 : want) : sms * 16ll);
  zero_skipped_rows_kernel<<<blocks, 256, 0, s>>>(g, T, row_bytes, static_cast<uint8_t*>(out));
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
  return align256(4 * sizeof(long long)) + align256(sizeof(int) * n_groups) +
         align256(sizeof(int) * n_seq) + align256(sizeof(float2) * n_seq) +
         align256(sizeof(float2) * n_seq) + align256(sizeof(int) * n_seq) +
         align256(sizeof(LossSums) * kLossFinalMaxBlocks);
}

LossWs carve_loss_ws(void* ws, int n_seq, int n_groups) {
  char* p = static_cast<char*>(ws);
  LossWs w;
  w.scal = reinterpret_cast<unsigned long long*>(p);  // cleared with gsize in one memset
  p += align256(4 * sizeof(long long));
  w.gsize = reinterpret_cast<int*>(p);
  p += align256(sizeof(int) * n_groups);
  w.n_tok = reinterpret_cast<int*>(p);
  p += align256(sizeof(int) * n_seq);
  w.part_l = reinterpret_cast<float2*>(p);
  p += align256(sizeof(float2) * n_seq);
  w.part_rk = reinterpret_cast<float2*>(p);
  p += align256(sizeof(float2) * n_seq);
  w.part_clip = reinterpret_cast<int*>(p);
  p += align256(sizeof(int) * n_seq);
  w.bpart = p;
  return w;
}

// Resident blocks per SM of a kernel (a property of the kernel and the
// architecture), looked up once per kernel; racing first calls store the same value.
template <class K>
int resident_blocks(K kernel, std::atomic<int>& cache) {
  int res = cache.load(std::memory_order_relaxed);
  if (res == 0) {
    int r = 0;
    res = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&r, kernel, kLossThreads, 0) == cudaSuccess &&
                  r > 0
              ? r
              : 1;
    cache.store(res, std::memory_order_relaxed);
  }
  return res;
}

cudaError_t launch_policy_loss(const float* logp, const float* old_logp, const float* ref_logp,
                               const float* adv, const int* cu_seqlens, const int* group_id,
                               int n_seq, int n_groups, const uint8_t* loss_mask, long long T,
                               float clip_eps, float kl_beta, int agg, float* loss, float* g,
                               float* stats, const LossWs& w, cudaStream_t s, int* err,
                               const float* cscale, const float* rewards, int std_mode,
                               float adv_eps, float* adv_out) {
  // scal (groups, tokens, ticket, barrier) and gsize are adjacent: one clear
  cudaError_t e = cudaMemsetAsync(w.scal, 0,
                                  reinterpret_cast<char*>(w.gsize + n_groups) -
                                      reinterpret_cast<char*>(w.scal), s);
  if (e != cudaSuccess) return e;
  const int sms = sm_count();
  // a group of 16 lanes per sequence when they are short, else a warp
  const bool short_seqs = T <= 128ll * n_seq;
  const bool with_adv = rewards != nullptr;
  // the final sum's chunks depend only on n_seq (fixed order on any device)
  const int chunk = max(256, (n_seq + kLossFinalMaxBlocks - 1) / kLossFinalMaxBlocks);
  const int nb = (n_seq + chunk - 1) / chunk;
  const int per_block = (kLossThreads / 32) * (short_seqs ? 2 : 1);  // sequences in flight per block
  const long long seq_blocks = (n_seq + per_block - 1) / per_block;
  const long long group_blocks =
      with_adv ? (static_cast<long long>(n_groups) + kLossThreads / 32 - 1) / (kLossThreads / 32) : 1;
  const long long count_blocks = agg == 1 ? max(1ll, min(T / 16 / kLossThreads, 4ll * sms)) : 1;

  LossLaunch a;
  a.logp = logp;
  a.old_logp = old_logp;
  a.ref_logp = ref_logp;
  a.adv = with_adv ? adv_out : adv;
  a.adv_out = adv_out;
  a.rewards = rewards;
  a.std_mode = std_mode;
  a.adv_eps = adv_eps;
  a.cu = cu_seqlens;
  a.gid = group_id;
  a.n_seq = n_seq;
  a.n_groups = n_groups;
  a.lm = loss_mask;
  a.clip_eps = clip_eps;
  a.kl_beta = kl_beta;
  a.agg = agg;
  a.cscale = cscale;
  a.loss = loss;
  a.g = g;
  a.stats = stats;
  a.w = w;
  a.chunk = chunk;
  a.nb = nb;
  a.err = err;

  if (n_seq <= kLossFusedMaxSeq) {
    // one cooperative launch: enough blocks for each phase, never more than
    // can be resident at once (every phase strides over the grid)
    using Kernel = void (*)(const LossLaunch);
    static const Kernel kernels[4] = {loss_fused_kernel<16, false>, loss_fused_kernel<32, false>,
                                      loss_fused_kernel<16, true>, loss_fused_kernel<32, true>};
    static std::atomic<int> resident[4] = {{0}, {0}, {0}, {0}};
    const int variant = (short_seqs ? 0 : 1) + (with_adv ? 2 : 0);
    const int res = resident_blocks(kernels[variant], resident[variant]);
    const long long want =
        max(max(seq_blocks, group_blocks), max(static_cast<long long>(nb), count_blocks));
    const int grid = static_cast<int>(max(1ll, min(want, static_cast<long long>(sms) * res)));
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(grid), 1, 1);
    cfg.blockDim = dim3(kLossThreads, 1, 1);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, kernels[variant], a);
    note_launches(1);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
  }
  // three launches
  const int cblocks = static_cast<int>(max(1ll, min(max(max(group_blocks, count_blocks),
                                                        (n_seq + kLossThreads - 1ll) / kLossThreads),
                                                    4ll * sms)));
  if (with_adv)
    loss_counts_kernel<true><<<cblocks, kLossThreads, 0, s>>>(a);
  else
    loss_counts_kernel<false><<<cblocks, kLossThreads, 0, s>>>(a);
  static std::atomic<int> resident_tok[2] = {{0}, {0}};
  const int res = short_seqs ? resident_blocks(loss_token_kernel<16>, resident_tok[0])
                             : resident_blocks(loss_token_kernel<32>, resident_tok[1]);
  const int tblocks = static_cast<int>(max(1ll, min(seq_blocks, static_cast<long long>(sms) * res)));
  if (short_seqs)
    loss_token_kernel<16><<<tblocks, kLossThreads, 0, s>>>(a);
  else
    loss_token_kernel<32><<<tblocks, kLossThreads, 0, s>>>(a);
  loss_final_kernel<<<nb, kLossThreads, 0, s>>>(a);
  note_launches(3);
  return cudaGetLastError();
}

}  // namespace spo
