// ranker.cu -- the offline structural ranker of CUDAPerf: z-scored 11-feature
// vectors through an 11 -> 64 -> 32 -> 1 ReLU MLP (s_psi), and the pairwise
// logistic ranking loss mean softplus(-(s(y+) - s(y-))) with its gradient
// with respect to every MLP parameter.
//
// One warp evaluates one program (scores) or one pair (loss).  Lane l owns
// hidden units l and l + 32 of layer 1 and unit l of layer 2, so it also owns
// the gradient rows of those units and accumulates them in registers over
// the pairs its warp visits, in a fixed order: results are deterministic.
#include <math.h>

#include "internal.h"

namespace spo {

namespace {

constexpr int kF = kRankerFeatures;  // 11
constexpr int kH1 = 64, kH2 = 32;
constexpr int kW2Stride = kH1 + 1;  // padded row: conflict-free row and column reads
// offsets in the packed parameter vector
constexpr int oW1 = 0, oB1 = oW1 + kH1 * kF, oW2 = oB1 + kH1, oB2 = oW2 + kH2 * kH1,
              oW3 = oB2 + kH2, oB3 = oW3 + kH2;
static_assert(oB3 + 1 == kRankerParams, "packed layout");
constexpr int kWarps = 8;

struct Smem {
  float W1[kH1 * kF];
  float b1[kH1];
  float W2[kH2 * kW2Stride];
  float b2[kH2];
  float w3[kH2];
  float b3;
  float mu[kF];
  float inv_sigma[kF];
};

__device__ void load_params(Smem& sm, const float* prm, const float* mu, const float* sigma) {
  for (int i = threadIdx.x; i < kH1 * kF; i += blockDim.x) sm.W1[i] = prm[oW1 + i];
  for (int i = threadIdx.x; i < kH1; i += blockDim.x) sm.b1[i] = prm[oB1 + i];
  for (int i = threadIdx.x; i < kH2 * kH1; i += blockDim.x)
    sm.W2[(i / kH1) * kW2Stride + i % kH1] = prm[oW2 + i];
  for (int i = threadIdx.x; i < kH2; i += blockDim.x) {
    sm.b2[i] = prm[oB2 + i];
    sm.w3[i] = prm[oW3 + i];
  }
  for (int i = threadIdx.x; i < kF; i += blockDim.x) {
    sm.mu[i] = mu[i];
    sm.inv_sigma[i] = 1.f / sigma[i];
  }
  if (threadIdx.x == 0) sm.b3 = prm[oB3];
  __syncthreads();
}

struct Act {  // this lane's share of one forward pass
  float x[kF];        // z-scored features (every lane holds all 11)
  float a1lo, a1hi;   // pre-activations of units lane, lane + 32
  float h1lo, h1hi;   // post-activation (after dropout)
  float a2, h2;       // unit lane of layer 2
  float s;            // score (warp-uniform)
};

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// keep1 / keep2: this member's dropout keep flags (NULL: no dropout), scale = 1 / (1 - p).
__device__ void forward(const Smem& sm, const float* phi_row, const uint8_t* keep1,
                        const uint8_t* keep2, float scale, int lane, Act& a) {
#pragma unroll
  for (int i = 0; i < kF; ++i) a.x[i] = (phi_row[i] - sm.mu[i]) * sm.inv_sigma[i];
  float lo = sm.b1[lane], hi = sm.b1[lane + 32];
#pragma unroll
  for (int i = 0; i < kF; ++i) {
    lo = fmaf(sm.W1[lane * kF + i], a.x[i], lo);
    hi = fmaf(sm.W1[(lane + 32) * kF + i], a.x[i], hi);
  }
  a.a1lo = lo;
  a.a1hi = hi;
  a.h1lo = fmaxf(lo, 0.f);
  a.h1hi = fmaxf(hi, 0.f);
  if (keep1) {
    a.h1lo *= keep1[lane] ? scale : 0.f;
    a.h1hi *= keep1[lane + 32] ? scale : 0.f;
  }
  float z = sm.b2[lane];
  const float* w2 = sm.W2 + lane * kW2Stride;
#pragma unroll
  for (int k = 0; k < 32; ++k) {
    z = fmaf(w2[k], __shfl_sync(0xffffffffu, a.h1lo, k), z);
    z = fmaf(w2[k + 32], __shfl_sync(0xffffffffu, a.h1hi, k), z);
  }
  a.a2 = z;
  a.h2 = fmaxf(z, 0.f);
  if (keep2) a.h2 *= keep2[lane] ? scale : 0.f;
  a.s = warp_sum(sm.w3[lane] * a.h2) + sm.b3;
}

struct Grad {  // this lane's gradient rows
  float W1lo[kF], W1hi[kF];
  float b1lo, b1hi;
  float W2[kH1];
  float b2, w3, b3;
};

__device__ void backward(const Smem& sm, const Act& a, const uint8_t* keep1, const uint8_t* keep2,
                         float scale, float ds, int lane, Grad& g) {
  g.w3 = fmaf(a.h2, ds, g.w3);
  if (lane == 0) g.b3 += ds;
  float dh2 = sm.w3[lane] * ds;
  if (keep2) dh2 *= keep2[lane] ? scale : 0.f;
  const float da2 = a.a2 > 0.f ? dh2 : 0.f;
  g.b2 += da2;
#pragma unroll
  for (int k = 0; k < 32; ++k) {
    g.W2[k] = fmaf(da2, __shfl_sync(0xffffffffu, a.h1lo, k), g.W2[k]);
    g.W2[k + 32] = fmaf(da2, __shfl_sync(0xffffffffu, a.h1hi, k), g.W2[k + 32]);
  }
  // dh1[k] = sum_j W2[j][k] da2[j] for k = lane, lane + 32
  float dlo = 0.f, dhi = 0.f;
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    const float d = __shfl_sync(0xffffffffu, da2, j);
    dlo = fmaf(sm.W2[j * kW2Stride + lane], d, dlo);
    dhi = fmaf(sm.W2[j * kW2Stride + lane + 32], d, dhi);
  }
  if (keep1) {
    dlo *= keep1[lane] ? scale : 0.f;
    dhi *= keep1[lane + 32] ? scale : 0.f;
  }
  const float da1lo = a.a1lo > 0.f ? dlo : 0.f;
  const float da1hi = a.a1hi > 0.f ? dhi : 0.f;
  g.b1lo += da1lo;
  g.b1hi += da1hi;
#pragma unroll
  for (int i = 0; i < kF; ++i) {
    g.W1lo[i] = fmaf(da1lo, a.x[i], g.W1lo[i]);
    g.W1hi[i] = fmaf(da1hi, a.x[i], g.W1hi[i]);
  }
}

__global__ void __launch_bounds__(kWarps * 32) ranker_scores_kernel(
    const float* phi, const float* mu, const float* sigma, int n, const float* prm, float* scores) {
  __shared__ Smem sm;
  load_params(sm, prm, mu, sigma);
  const int lane = threadIdx.x & 31;
  const int w0 = blockIdx.x * kWarps + (threadIdx.x >> 5);
  for (int r = w0; r < n; r += gridDim.x * kWarps) {
    Act a;
    forward(sm, phi + static_cast<size_t>(r) * kF, nullptr, nullptr, 1.f, lane, a);
    if (lane == 0) scores[r] = a.s;
  }
}

// Per-block partials: [gridDim.x][kRankerParams + 1] (last entry: sum of softplus).
__global__ void __launch_bounds__(kWarps * 32) ranker_pair_kernel(
    const float* phi, const float* mu, const float* sigma, const int* pos, const int* neg,
    int n_pairs, const float* prm, const uint8_t* keep1, const uint8_t* keep2, float drop_p,
    float* block_part) {
  __shared__ Smem sm;
  __shared__ float red[kRankerParams + 1];
  for (int i = threadIdx.x; i <= kRankerParams; i += blockDim.x) red[i] = 0.f;
  load_params(sm, prm, mu, sigma);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const float scale = 1.f / (1.f - drop_p);
  const float inv_p = 1.f / static_cast<float>(n_pairs);
  Grad g = {};
  float lsum = 0.f;
  for (int k = blockIdx.x * kWarps + warp; k < n_pairs; k += gridDim.x * kWarps) {
    const uint8_t* k1p = keep1 ? keep1 + static_cast<size_t>(k) * 2 * kH1 : nullptr;
    const uint8_t* k1n = keep1 ? k1p + kH1 : nullptr;
    const uint8_t* k2p = keep2 ? keep2 + static_cast<size_t>(k) * 2 * kH2 : nullptr;
    const uint8_t* k2n = keep2 ? k2p + kH2 : nullptr;
    Act ap, an;
    forward(sm, phi + static_cast<size_t>(pos[k]) * kF, k1p, k2p, scale, lane, ap);
    forward(sm, phi + static_cast<size_t>(neg[k]) * kF, k1n, k2n, scale, lane, an);
    const float delta = ap.s - an.s;
    // softplus(-delta) = max(-delta, 0) + log1p(exp(-|delta|))
    lsum += fmaxf(-delta, 0.f) + log1pf(expf(-fabsf(delta)));
    const float dd = -inv_p / (1.f + expf(delta));  // dL/d delta
    backward(sm, ap, k1p, k2p, scale, dd, lane, g);
    backward(sm, an, k1n, k2n, scale, -dd, lane, g);
  }
  // add the warps' rows into the block's slot one warp at a time (fixed order);
  // within a warp every lane owns distinct entries
  for (int w = 0; w < kWarps; ++w) {
    if (warp == w) {
#pragma unroll
      for (int i = 0; i < kF; ++i) {
        red[oW1 + lane * kF + i] += g.W1lo[i];
        red[oW1 + (lane + 32) * kF + i] += g.W1hi[i];
      }
      red[oB1 + lane] += g.b1lo;
      red[oB1 + lane + 32] += g.b1hi;
#pragma unroll
      for (int k = 0; k < kH1; ++k) red[oW2 + lane * kH1 + k] += g.W2[k];
      red[oB2 + lane] += g.b2;
      red[oW3 + lane] += g.w3;
      if (lane == 0) {
        red[oB3] += g.b3;
        red[kRankerParams] += lsum;
      }
    }
    __syncthreads();
  }
  float* out = block_part + static_cast<size_t>(blockIdx.x) * (kRankerParams + 1);
  for (int i = threadIdx.x; i <= kRankerParams; i += blockDim.x) out[i] = red[i];
}

// Fixed-order sum of the per-block partials -> grad and loss.
__global__ void ranker_reduce_kernel(const float* block_part, int n_blocks, int n_pairs,
                                     float* grad, float* loss) {
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i <= kRankerParams; i += gridDim.x * blockDim.x) {
    double v = 0.0;
    for (int b = 0; b < n_blocks; ++b) v += block_part[static_cast<size_t>(b) * (kRankerParams + 1) + i];
    if (i < kRankerParams) {
      if (grad) grad[i] = static_cast<float>(v);
    } else {
      *loss = static_cast<float>(v / n_pairs);
    }
  }
}



}  // namespace

int ranker_blocks(int n_pairs) {
  const int want = (n_pairs + kWarps - 1) / kWarps;
  const int cap = 2 * sm_count();
  return want < 1 ? 1 : (want < cap ? want : cap);
}

size_t ranker_ws_bytes(int n_pairs) {
  return static_cast<size_t>(ranker_blocks(n_pairs)) * (kRankerParams + 1) * sizeof(float);
}

cudaError_t launch_ranker_scores(const float* phi, const float* mu, const float* sigma, int n,
                                 const float* params, float* scores, cudaStream_t s) {
  const int want = (n + kWarps - 1) / kWarps;
  const int cap = 8 * sm_count();
  ranker_scores_kernel<<<want < cap ? want : cap, kWarps * 32, 0, s>>>(phi, mu, sigma, n, params,
                                                                       scores);
  note_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_ranker_pair_loss(const float* phi, const float* mu, const float* sigma,
                                    const int* pos, const int* neg, int n_pairs,
                                    const float* params, const uint8_t* keep1,
                                    const uint8_t* keep2, float drop_p, float* loss, float* grad,
                                    float* ws, cudaStream_t s) {
  const int nb = ranker_blocks(n_pairs);
  ranker_pair_kernel<<<nb, kWarps * 32, 0, s>>>(phi, mu, sigma, pos, neg, n_pairs, params, keep1,
                                                keep2, drop_p, ws);
  ranker_reduce_kernel<<<(kRankerParams + 256) / 256, 256, 0, s>>>(ws, nb, n_pairs, grad, loss);
  note_launches(2);
  return cudaGetLastError();
}

}  // namespace spo
