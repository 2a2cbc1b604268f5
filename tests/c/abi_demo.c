/* abi_demo.c -- uses libspo from plain C99 (no Python, no C++): allocates
 * its own device buffers, runs the whole path once on a small batch, and
 * checks closed forms that need no reference implementation:
 *   - with H = 0 every logit is 0, so logp = -ln V and entropy = ln V;
 *   - log-probs are <= 0 and the loss is finite;
 *   - every status is SPO_OK and no device wait expired;
 *   - the one-call step (spo_grpo_step, workspace from spo_workspace_size)
 *     gives the same bits as the separate calls, and a bad argument is
 *     reported through spo_last_error_detail.
 * Build: cc -std=c99 abi_demo.c -I include -I <cuda>/include -L <lib> -lspo
 *        -L <cuda>/lib64 -lcudart -Wl,-rpath,<lib>
 * Exit status 0 on success. */
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <cuda_runtime_api.h>

#include "spo.h"

#define T 64
#define D 128
#define V 1024
#define NSEQ 8
#define NGROUPS 2

static int check(spo_status st, const char* what) {
  if (st != SPO_OK) {
    char buf[256];
    spo_last_error(buf, sizeof(buf));
    fprintf(stderr, "%s failed: %s (%s)\n", what, spo_status_string(st), buf);
    return 1;
  }
  return 0;
}

static void* dev_alloc(size_t n) {
  void* p = NULL;
  if (cudaMalloc(&p, n) != cudaSuccess) {
    fprintf(stderr, "cudaMalloc(%zu) failed\n", n);
    exit(2);
  }
  return p;
}

static void* dev_copy(const void* h, size_t n) {
  void* p = dev_alloc(n);
  cudaMemcpy(p, h, n, cudaMemcpyHostToDevice);
  return p;
}

int main(void) {
  static uint16_t h_H[T * D];     /* bf16 zeros: uniform logits */
  static uint16_t h_W[V * D];
  int32_t h_tgt[T], h_cu[NSEQ + 1], h_gid[NSEQ];
  float h_rew[NSEQ], h_old[T];
  uint8_t h_mask[T];
  uint32_t s = 12345u;
  int i, bad = 0;
  memset(h_H, 0, sizeof(h_H));
  for (i = 0; i < V * D; ++i) {  /* small bf16 weights: 0x3c00 + jitter ~ 0.0078 .. 0.0156 */
    s = s * 1664525u + 1013904223u;
    h_W[i] = (uint16_t)(0x3c00u + ((s >> 24) & 0x7fu)) | (uint16_t)((s & 1u) << 15);
  }
  for (i = 0; i < T; ++i) {
    s = s * 1664525u + 1013904223u;
    h_tgt[i] = (int32_t)((s >> 8) % V);
    h_mask[i] = 1;
    h_old[i] = -logf((float)V) + 0.01f * (float)((int)(s & 7u) - 3);
  }
  for (i = 0; i <= NSEQ; ++i) h_cu[i] = i * (T / NSEQ);
  for (i = 0; i < NSEQ; ++i) {
    h_gid[i] = i % NGROUPS;
    h_rew[i] = 0.25f * (float)i;
  }

  void* H = dev_copy(h_H, sizeof(h_H));
  void* W = dev_copy(h_W, sizeof(h_W));
  int32_t* tgt = (int32_t*)dev_copy(h_tgt, sizeof(h_tgt));
  int32_t* cu = (int32_t*)dev_copy(h_cu, sizeof(h_cu));
  int32_t* gid = (int32_t*)dev_copy(h_gid, sizeof(h_gid));
  float* rew = (float*)dev_copy(h_rew, sizeof(h_rew));
  float* old = (float*)dev_copy(h_old, sizeof(h_old));
  uint8_t* mask = (uint8_t*)dev_copy(h_mask, sizeof(h_mask));
  uint8_t* lm = (uint8_t*)dev_alloc(T);
  int32_t* ntok = (int32_t*)dev_alloc(NSEQ * sizeof(int32_t));
  float* logp = (float*)dev_alloc(T * sizeof(float));
  float* ent = (float*)dev_alloc(T * sizeof(float));
  float* lse = (float*)dev_alloc(T * sizeof(float));
  float* adv = (float*)dev_alloc(NSEQ * sizeof(float));
  float* loss = (float*)dev_alloc(sizeof(float));
  float* g = (float*)dev_alloc(T * sizeof(float));
  void* dH = dev_alloc((size_t)T * D * 2);
  float* dW = (float*)dev_alloc((size_t)V * D * sizeof(float));
  size_t ws_f = 0, ws_l = 0, ws_b = 0;
  if (check(spo_logprobs_workspace_size(T, D, V, &ws_f), "logprobs ws") ||
      check(spo_policy_loss_workspace_size(NSEQ, NGROUPS, &ws_l), "loss ws") ||
      check(spo_policy_loss_bwd_workspace_size(T, D, V, &ws_b), "bwd ws"))
    return 1;
  void* wf = dev_alloc(ws_f);
  void* wl = dev_alloc(ws_l);
  void* wb = dev_alloc(ws_b);

  if (check(spo_token_select(cu, mask, tgt, NSEQ, T, 1024, lm, ntok, NULL), "token_select") ||
      check(spo_logprobs_fwd(H, W, tgt, lm, T, D, V, 1.0f, logp, ent, lse, wf, ws_f, NULL),
            "logprobs_fwd") ||
      check(spo_group_advantages(rew, gid, NSEQ, NGROUPS, SPO_STD_UNBIASED, 1e-6f, adv, NULL),
            "group_advantages") ||
      check(spo_policy_loss_fwd(logp, old, NULL, adv, cu, gid, NSEQ, NGROUPS, lm, T, 0.2f, 0.0f,
                                SPO_AGG_SEQ_GROUP, loss, g, NULL, wl, ws_l, NULL),
            "policy_loss_fwd") ||
      check(spo_policy_loss_bwd(H, W, tgt, lse, g, T, D, V, 1.0f, dH, dW, 0, wb, ws_b, NULL),
            "policy_loss_bwd"))
    return 1;
  int code = 0;
  if (check(spo_device_error(&code, NULL), "device_error")) return 1;

  /* the same step as one call, with one workspace sized for the whole step */
  size_t ws_all = 0;
  if (check(spo_workspace_size(T, D, V, NSEQ, &ws_all), "workspace_size")) return 1;
  void* wall = dev_alloc(ws_all);
  float* loss2 = (float*)dev_alloc(sizeof(float));
  float* logp2 = (float*)dev_alloc(T * sizeof(float));
  float* dW2 = (float*)dev_alloc((size_t)V * D * sizeof(float));
  spo_grpo_batch batch = {H, W, tgt, mask, cu, gid, rew, old, NULL, T, D, V, NSEQ, NGROUPS};
  spo_grpo_params prm = {1.0f, 1024, 0.2f, 0.0f, SPO_AGG_SEQ_GROUP, SPO_STD_UNBIASED, 1e-6f, NULL};
  spo_grpo_outputs out;
  memset(&out, 0, sizeof(out));
  out.loss = loss2;
  out.logp = logp2;
  out.dW = dW2;
  if (check(spo_grpo_step(&batch, &prm, &out, NULL, wall, ws_all, NULL), "grpo_step") ||
      check(spo_sync_check(NULL), "sync_check"))
    return 1;
  /* an argument error is reported, with its text, under the boundary's name */
  char why[256];
  if (spo_grpo_step(NULL, &prm, &out, NULL, wall, ws_all, NULL) != SPO_ERR_INVALID_ARG ||
      spo_last_error_detail(why, sizeof(why)) != SPO_ERR_INVALID_ARG || why[0] == '\0')
    ++bad;

  float h_logp[T], h_ent[T], h_loss;
  cudaMemcpy(h_logp, logp, sizeof(h_logp), cudaMemcpyDeviceToHost);
  cudaMemcpy(h_ent, ent, sizeof(h_ent), cudaMemcpyDeviceToHost);
  cudaMemcpy(&h_loss, loss, sizeof(float), cudaMemcpyDeviceToHost);
  const float lnV = logf((float)V);
  for (i = 0; i < T; ++i) {
    if (fabsf(h_logp[i] + lnV) > 1e-4f || fabsf(h_ent[i] - lnV) > 1e-4f) ++bad;
  }
  if (!isfinite(h_loss)) ++bad;
  {
    /* g has no zero on the loss tokens here, so the one-call step gives the same bits */
    static float h_logp2[T], h_dW[64], h_dW2[64];
    float h_loss2;
    cudaMemcpy(h_logp2, logp2, sizeof(h_logp2), cudaMemcpyDeviceToHost);
    cudaMemcpy(&h_loss2, loss2, sizeof(float), cudaMemcpyDeviceToHost);
    cudaMemcpy(h_dW, dW, sizeof(h_dW), cudaMemcpyDeviceToHost);
    cudaMemcpy(h_dW2, dW2, sizeof(h_dW2), cudaMemcpyDeviceToHost);
    if (memcmp(h_logp, h_logp2, sizeof(h_logp2)) != 0 || memcmp(&h_loss, &h_loss2, sizeof(float)) != 0 ||
        memcmp(h_dW, h_dW2, sizeof(h_dW)) != 0)
      ++bad;
  }
  printf("libspo %d.%d from C: logp[0]=%.6f (-ln V=%.6f) entropy[0]=%.6f loss=%.6g bad=%d\n",
         spo_version() >> 16, spo_version() & 0xffff, h_logp[0], -lnV, h_ent[0], h_loss, bad);
  return bad ? 1 : 0;
}
