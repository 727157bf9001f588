/* A plain C caller of libavits.so (include/avits.h): device buffers from the
 * CUDA runtime, the temporal score and the fused selection through the C ABI,
 * results checked against host computations in this file.  Built and run by
 * tests/test_c_abi.py on a GPU; prints "ok" and exits 0 on success. */
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <cuda_runtime.h>

#include "avits.h"

#define CHECK_CUDA(x)                                                             \
  do {                                                                            \
    cudaError_t e_ = (x);                                                         \
    if (e_ != cudaSuccess) {                                                      \
      fprintf(stderr, "CUDA error %s at line %d\n", cudaGetErrorString(e_), __LINE__); \
      return 2;                                                                   \
    }                                                                             \
  } while (0)

#define CHECK_AVITS(x)                                                            \
  do {                                                                            \
    avits_status s_ = (x);                                                        \
    if (s_ != AVITS_OK) {                                                         \
      fprintf(stderr, "avits error %s at line %d\n", avits_status_string(s_), __LINE__); \
      return 3;                                                                   \
    }                                                                             \
  } while (0)

/* xorshift32: a reproducible host pattern */
static uint32_t rng_state = 12345u;
static float next_unit(void) {
  rng_state ^= rng_state << 13;
  rng_state ^= rng_state >> 17;
  rng_state ^= rng_state << 5;
  return (float)(rng_state >> 8) / 16777216.0f;
}

/* the selection order: S descending, index ascending */
static const float* g_S;
static int cmp_desc(const void* a, const void* b) {
  const int i = *(const int*)a, j = *(const int*)b;
  if (g_S[i] > g_S[j]) return -1;
  if (g_S[i] < g_S[j]) return 1;
  return (i > j) - (i < j);
}

int main(void) {
  enum { N = 300, D = 96, M = 1000, K = 123 };
  /* --- temporal score: V_i = ||h_t - h_prev|| / (||h_prev|| + eps) --- */
  float* ht = (float*)malloc(sizeof(float) * N * D);
  float* hp = (float*)malloc(sizeof(float) * N * D);
  for (int i = 0; i < N * D; ++i) {
    hp[i] = next_unit() - 0.5f;
    ht[i] = hp[i] + 0.1f * (next_unit() - 0.5f);
  }
  float *d_ht, *d_hp, *d_V;
  CHECK_CUDA(cudaMalloc((void**)&d_ht, sizeof(float) * N * D));
  CHECK_CUDA(cudaMalloc((void**)&d_hp, sizeof(float) * N * D));
  CHECK_CUDA(cudaMalloc((void**)&d_V, sizeof(float) * N));
  CHECK_CUDA(cudaMemcpy(d_ht, ht, sizeof(float) * N * D, cudaMemcpyHostToDevice));
  CHECK_CUDA(cudaMemcpy(d_hp, hp, sizeof(float) * N * D, cudaMemcpyHostToDevice));
  CHECK_AVITS(avits_score_temporal(d_ht, d_hp, AVITS_F32, 1, N, D, 1e-6f, d_V, NULL));
  CHECK_AVITS(avits_device_status(NULL));
  float V[N];
  CHECK_CUDA(cudaMemcpy(V, d_V, sizeof(V), cudaMemcpyDeviceToHost));
  for (int i = 0; i < N; ++i) {
    double dd = 0.0, pp = 0.0;
    for (int c = 0; c < D; ++c) {
      const double d = (double)ht[i * D + c] - (double)hp[i * D + c];
      dd += d * d;
      pp += (double)hp[i * D + c] * hp[i * D + c];
    }
    const double ref = sqrt(dd) / (sqrt(pp) + 1e-6);
    if (fabs(V[i] - ref) > 1e-5 * ref + 1e-7) {
      fprintf(stderr, "V[%d] = %.8g, host %.8g\n", i, V[i], ref);
      return 4;
    }
  }

  /* --- fused selection: S = a*A^ + (1-a)*V^, top-K, ties by lower index --- */
  float* A = (float*)malloc(sizeof(float) * M);
  float* W = (float*)malloc(sizeof(float) * M);
  for (int i = 0; i < M; ++i) {
    A[i] = (float)((int)(next_unit() * 64.0f)) / 64.0f;   /* coarse values: ties */
    W[i] = next_unit();
  }
  float *d_A, *d_W, *d_S;
  int32_t *d_sel, *d_off;
  uint8_t* d_mask;
  CHECK_CUDA(cudaMalloc((void**)&d_A, sizeof(float) * M));
  CHECK_CUDA(cudaMalloc((void**)&d_W, sizeof(float) * M));
  CHECK_CUDA(cudaMalloc((void**)&d_S, sizeof(float) * M));
  CHECK_CUDA(cudaMalloc((void**)&d_sel, sizeof(int32_t) * K));
  CHECK_CUDA(cudaMalloc((void**)&d_off, sizeof(int32_t) * M));
  CHECK_CUDA(cudaMalloc((void**)&d_mask, M));
  CHECK_CUDA(cudaMemcpy(d_A, A, sizeof(float) * M, cudaMemcpyHostToDevice));
  CHECK_CUDA(cudaMemcpy(d_W, W, sizeof(float) * M, cudaMemcpyHostToDevice));
  CHECK_AVITS(avits_fuse_select(d_A, d_W, 1, M, 0.5f, 1e-6f, K, d_S, d_sel, d_mask, d_off, NULL));
  CHECK_AVITS(avits_device_status(NULL));
  float S[M];
  int32_t sel[K], off[M];
  uint8_t mask[M];
  CHECK_CUDA(cudaMemcpy(S, d_S, sizeof(S), cudaMemcpyDeviceToHost));
  CHECK_CUDA(cudaMemcpy(sel, d_sel, sizeof(sel), cudaMemcpyDeviceToHost));
  CHECK_CUDA(cudaMemcpy(off, d_off, sizeof(off), cudaMemcpyDeviceToHost));
  CHECK_CUDA(cudaMemcpy(mask, d_mask, sizeof(mask), cudaMemcpyDeviceToHost));
  /* host S in the same fp32 operation order (min, max, (x-min)/den, a*x+b*y) */
  float amn = A[0], amx = A[0], vmn = W[0], vmx = W[0];
  for (int i = 1; i < M; ++i) {
    if (A[i] < amn) amn = A[i];
    if (A[i] > amx) amx = A[i];
    if (W[i] < vmn) vmn = W[i];
    if (W[i] > vmx) vmx = W[i];
  }
  volatile float aden = amx - amn;
  aden = aden + 1e-6f;
  volatile float vden = vmx - vmn;
  vden = vden + 1e-6f;
  float Sh[M];
  for (int i = 0; i < M; ++i) {
    volatile float an = A[i] - amn;
    an = an / aden;
    volatile float vn = W[i] - vmn;
    vn = vn / vden;
    volatile float t1 = 0.5f * an;
    volatile float t2 = 0.5f * vn;
    Sh[i] = t1 + t2;
    if (memcmp(&Sh[i], &S[i], sizeof(float)) != 0) {
      fprintf(stderr, "S[%d] = %.9g, host %.9g\n", i, S[i], Sh[i]);
      return 5;
    }
  }
  int order[M];
  for (int i = 0; i < M; ++i) order[i] = i;
  g_S = Sh;
  qsort(order, M, sizeof(int), cmp_desc);
  uint8_t want[M];
  memset(want, 0, sizeof(want));
  for (int j = 0; j < K; ++j) want[order[j]] = 1;
  int c = 0;
  for (int i = 0; i < M; ++i) {
    if (mask[i] != want[i] || off[i] != i + 3 * c) {
      fprintf(stderr, "token %d: mask %d (host %d), offset %d (host %d)\n", i, mask[i], want[i],
              off[i], i + 3 * c);
      return 6;
    }
    if (want[i]) {
      if (sel[c] != i) {
        fprintf(stderr, "sel[%d] = %d, host %d\n", c, sel[c], i);
        return 7;
      }
      ++c;
    }
  }
  printf("ok\n");
  return 0;
}
