/*
 * Test helper: a plain C99 program that uses the ES library only through
 * include/esopt.h and the CUDA runtime's C API (no Python, no C++). It reads
 * n and n bf16 bit patterns (decimal) from stdin, puts them in device memory,
 * and runs:
 *   P: es_perturb(seed 11, sigma 1e-3)
 *   R: es_restore(seed 11, sigma 1e-3)
 *   U: es_update(seeds {3, 5, 7}, coeffs {1e-4, -2e-4, 5e-5})
 *   E: es_noise_fill(seed 11, index_base 0, n) into an fp32 buffer
 * printing each result as one line ("P v0 v1 ..."; bf16 as decimal bit
 * patterns, fp32 as %.9g). It also checks that a host pointer is refused
 * with ES_ERR_INVALID_ARG. Exits non-zero on any unexpected status.
 */
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>

#include <cuda_runtime_api.h>

#include "esopt.h"

static int expect(es_status_t st, es_status_t want, const char* what) {
  if (st != want) {
    fprintf(stderr, "%s: %s (%s), expected %s\n", what, es_status_string(st), es_last_error(),
            es_status_string(want));
    return 1;
  }
  return 0;
}

static int dump_bf16(const char* tag, const uint16_t* dev, uint16_t* host, uint64_t n) {
  uint64_t k;
  if (cudaMemcpy(host, dev, n * sizeof(uint16_t), cudaMemcpyDeviceToHost) != cudaSuccess) return 1;
  printf("%s", tag);
  for (k = 0; k < n; ++k) printf(" %u", (unsigned)host[k]);
  printf("\n");
  return 0;
}

int main(void) {
  unsigned long long n_in = 0;
  uint64_t n, k;
  uint16_t* host;
  float* host_eps;
  void* d_theta = NULL;
  float* d_eps = NULL;
  es_segment_t seg;
  es_plan_t plan = NULL;
  const uint64_t seeds[3] = {3u, 5u, 7u};
  const float coeffs[3] = {1e-4f, -2e-4f, 5e-5f};
  int rc = 0;

  if (scanf("%llu", &n_in) != 1 || n_in == 0) return 2;
  n = (uint64_t)n_in;
  host = (uint16_t*)malloc(n * sizeof(uint16_t));
  host_eps = (float*)malloc(n * sizeof(float));
  if (host == NULL || host_eps == NULL) return 2;
  for (k = 0; k < n; ++k) {
    unsigned v;
    if (scanf("%u", &v) != 1) return 2;
    host[k] = (uint16_t)v;
  }
  if (cudaMalloc(&d_theta, n * sizeof(uint16_t)) != cudaSuccess) return 3;
  if (cudaMalloc((void**)&d_eps, n * sizeof(float)) != cudaSuccess) return 3;
  if (cudaMemcpy(d_theta, host, n * sizeof(uint16_t), cudaMemcpyHostToDevice) != cudaSuccess)
    return 3;

  /* A host buffer is refused before any launch. */
  seg.data = host;
  seg.numel = n;
  seg.index_base = 0;
  rc |= expect(es_plan_create(&seg, 1, ES_BF16, &plan), ES_ERR_INVALID_ARG, "host segment");
  if (plan != NULL) rc = 1;

  seg.data = d_theta;
  rc |= expect(es_plan_create(&seg, 1, ES_BF16, &plan), ES_OK, "es_plan_create");
  if (rc) return 4;
  if (es_plan_numel(plan) != n) return 4;

  rc |= expect(es_perturb(plan, 11u, 1e-3f, NULL), ES_OK, "es_perturb");
  rc |= dump_bf16("P", (const uint16_t*)d_theta, host, n);
  rc |= expect(es_restore(plan, 11u, 1e-3f, NULL), ES_OK, "es_restore");
  rc |= dump_bf16("R", (const uint16_t*)d_theta, host, n);
  rc |= expect(es_update(plan, seeds, coeffs, 3, NULL), ES_OK, "es_update");
  rc |= dump_bf16("U", (const uint16_t*)d_theta, host, n);
  rc |= expect(es_noise_fill(11u, 0u, n, d_eps, NULL), ES_OK, "es_noise_fill");
  if (cudaMemcpy(host_eps, d_eps, n * sizeof(float), cudaMemcpyDeviceToHost) != cudaSuccess)
    rc = 1;
  printf("E");
  for (k = 0; k < n; ++k) printf(" %.9g", host_eps[k]);
  printf("\n");

  rc |= expect(es_plan_destroy(plan), ES_OK, "es_plan_destroy");
  cudaFree(d_theta);
  cudaFree(d_eps);
  free(host);
  free(host_eps);
  return rc;
}
