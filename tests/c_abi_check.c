/*
 * A plain C11 user of libgrpo.so (test infrastructure): checks that the
 * header compiles as C and that the library links and answers without any
 * Python in between.
 *
 *   c_abi_check host     sizing, status strings and host-side rejections
 *                        (no GPU needed); prints "ok" or the first failure
 *   c_abi_check device   Eq. 2 advantages and log-probs of a small fixed
 *                        batch on device memory from cudaMalloc; prints the
 *                        results, one value per line, for the caller to
 *                        compare with the float64 oracle
 */
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <cuda_runtime_api.h>

#include "grpo.h"

#define CHECK(cond)                                              \
  do {                                                           \
    if (!(cond)) {                                               \
      printf("FAILED line %d: %s\n", __LINE__, #cond);            \
      return 1;                                                  \
    }                                                            \
  } while (0)

static int host_checks(void) {
  const size_t full = grpo_workspace_bytes(32768, 4096, 155136, GRPO_WS_LOSS);
  CHECK(full > 0);
  CHECK(grpo_workspace_bytes_rows(32768, 20000, 4096, 155136, GRPO_WS_LOSS) < full);
  CHECK(grpo_workspace_bytes(10, 60, 100, GRPO_WS_LOSS) == 0);        /* Hd not a multiple of 64 */
  CHECK(strcmp(grpo_status_string(GRPO_OK), "GRPO_OK") == 0);
  CHECK(strcmp(grpo_status_string(GRPO_ERR_CAPACITY), "GRPO_ERR_CAPACITY") == 0);
  CHECK(grpo_vocab_chunk_cols(1000) == 1024);
  /* rejected on the host before any device work: G = 1, and a null output */
  float r[4] = {0, 1, 0, 1}, a[4];
  CHECK(grpo_group_advantages(r, 4, 1, 1e-6f, a, NULL) == GRPO_ERR_INVALID_ARG);
  CHECK(grpo_token_logprobs(NULL, NULL, NULL, NULL, 100, 64, 1000, NULL, NULL, 0, NULL) ==
        GRPO_ERR_INVALID_ARG);
  CHECK(grpo_check_device_status(NULL, NULL) == GRPO_ERR_INVALID_ARG);
  printf("ok\n");
  return 0;
}

/* bf16 bits of a float (round to nearest even; the inputs are finite) */
static uint16_t bf16(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  u += 0x7fffu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

static int device_run(void) {
  enum { G = 4, NR = 8, L = 40, T = NR * L, HD = 64, V = 300 };
  float rewards[NR] = {0, 1, 0.5f, 0, 1, 1, 0, 0.5f};
  static uint16_t H[T * HD], W[V * HD];
  static int32_t y[T];
  static uint8_t mask[T];
  /* a fixed pseudo-random batch (a linear congruential sequence) */
  uint32_t s = 12345u;
  for (int i = 0; i < T * HD; ++i) {
    s = s * 1664525u + 1013904223u;
    H[i] = bf16(((float)(s >> 8) / 16777216.0f - 0.5f) * 2.0f);
  }
  for (int i = 0; i < V * HD; ++i) {
    s = s * 1664525u + 1013904223u;
    W[i] = bf16(((float)(s >> 8) / 16777216.0f - 0.5f) * 0.5f);
  }
  for (int t = 0; t < T; ++t) {
    s = s * 1664525u + 1013904223u;
    y[t] = (int32_t)((s >> 8) % V);
    mask[t] = (uint8_t)((t % L) < 5 + (t / L) * 4);  /* response i has 5 + 4 i tokens */
  }
  void *dH, *dW, *dy, *dm, *dr, *da, *dl, *ws;
  const size_t ws_bytes = grpo_workspace_bytes(T, HD, V, GRPO_WS_LOGPROBS);
  CHECK(cudaMalloc(&dH, sizeof H) == cudaSuccess && cudaMalloc(&dW, sizeof W) == cudaSuccess);
  CHECK(cudaMalloc(&dy, sizeof y) == cudaSuccess && cudaMalloc(&dm, sizeof mask) == cudaSuccess);
  CHECK(cudaMalloc(&dr, sizeof rewards) == cudaSuccess && cudaMalloc(&da, sizeof rewards) == cudaSuccess);
  CHECK(cudaMalloc(&dl, T * sizeof(float)) == cudaSuccess && cudaMalloc(&ws, ws_bytes) == cudaSuccess);
  CHECK(cudaMemcpy(dH, H, sizeof H, cudaMemcpyHostToDevice) == cudaSuccess);
  CHECK(cudaMemcpy(dW, W, sizeof W, cudaMemcpyHostToDevice) == cudaSuccess);
  CHECK(cudaMemcpy(dy, y, sizeof y, cudaMemcpyHostToDevice) == cudaSuccess);
  CHECK(cudaMemcpy(dm, mask, sizeof mask, cudaMemcpyHostToDevice) == cudaSuccess);
  CHECK(cudaMemcpy(dr, rewards, sizeof rewards, cudaMemcpyHostToDevice) == cudaSuccess);
  CHECK(grpo_group_advantages((const float*)dr, NR, G, 1e-6f, (float*)da, NULL) == GRPO_OK);
  CHECK(grpo_token_logprobs((const uint16_t*)dH, (const uint16_t*)dW, (const int32_t*)dy,
                            (const uint8_t*)dm, T, HD, V, (float*)dl, ws, ws_bytes, NULL) == GRPO_OK);
  CHECK(grpo_check_device_status(ws, NULL) == GRPO_OK);
  float adv[NR], logp[T];
  CHECK(cudaMemcpy(adv, da, sizeof adv, cudaMemcpyDeviceToHost) == cudaSuccess);
  CHECK(cudaMemcpy(logp, dl, sizeof logp, cudaMemcpyDeviceToHost) == cudaSuccess);
  for (int i = 0; i < NR; ++i) printf("adv %.9g\n", adv[i]);
  for (int t = 0; t < T; ++t) printf("logp %.9g\n", logp[t]);
  /* the inputs, for the caller's oracle */
  for (int i = 0; i < T * HD; ++i) printf("H %u\n", (unsigned)H[i]);
  for (int i = 0; i < V * HD; ++i) printf("W %u\n", (unsigned)W[i]);
  for (int t = 0; t < T; ++t) printf("y %d %d\n", (int)y[t], (int)mask[t]);
  cudaFree(dH); cudaFree(dW); cudaFree(dy); cudaFree(dm); cudaFree(dr); cudaFree(da); cudaFree(dl); cudaFree(ws);
  return 0;
}

int main(int argc, char** argv) {
  if (argc > 1 && strcmp(argv[1], "device") == 0) return device_run();
  return host_checks();
}
