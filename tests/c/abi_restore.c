/*
 * abi_restore.c -- the C ABI used from plain C: a replica's state (bf16 and
 * fp32 tensors, one with a ragged tail, one misaligned by 4 bytes) is
 * fingerprinted, packed, damaged in transit, unpacked and verified, re-sent,
 * and compared by fingerprint diff; every step goes through flashrec.h, with
 * the CUDA runtime only for memory and streams.  Exits 0 on success, else
 * prints the failing check.
 */
#include <cuda_runtime.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include "flashrec.h"

#define CHECK_FR(x)                                                                        \
  do {                                                                                     \
    fr_status s_ = (x);                                                                    \
    if (s_ != FR_OK) {                                                                     \
      fprintf(stderr, "%s:%d %s -> %s (%s)\n", __FILE__, __LINE__, #x, fr_status_str(s_), \
              fr_last_error());                                                            \
      return 1;                                                                            \
    }                                                                                      \
  } while (0)
#define CHECK_CUDA(x)                                                                            \
  do {                                                                                           \
    cudaError_t e_ = (x);                                                                        \
    if (e_ != cudaSuccess) {                                                                     \
      fprintf(stderr, "%s:%d %s -> %s\n", __FILE__, __LINE__, #x, cudaGetErrorString(e_));       \
      return 1;                                                                                  \
    }                                                                                            \
  } while (0)
#define EXPECT(c)                                                   \
  do {                                                              \
    if (!(c)) {                                                     \
      fprintf(stderr, "%s:%d check failed: %s\n", __FILE__, __LINE__, #c); \
      return 1;                                                     \
    }                                                               \
  } while (0)

static uint64_t splitmix(uint64_t* s) {
  uint64_t z = (*s += 0x9E3779B97F4A7C15ull);
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

/* Random finite values in [-1, 1): fp32, and bf16 as the upper half of one. */
static float rand_unit(uint64_t* s) { return (float)((double)(splitmix(s) >> 11) / 9007199254740992.0 * 2.0 - 1.0); }

int main(void) {
  const uint64_t n_bf16 = 1000003, n_f32a = 700001, n_f32b = 300000;
  const uint64_t bytes[3] = {2 * n_bf16, 4 * n_f32a, 4 * n_f32b};
  const uint64_t off[3] = {0, 2000016, 4800036}; /* the third tensor starts 4 bytes past a 16-byte boundary */
  const uint64_t total = off[2] + bytes[2] + 16;
  const uint32_t dtypes[3] = {FR_DT_BF16, FR_DT_F32, FR_DT_F32};
  const uint64_t chunk = 64 * 1024;

  uint8_t* host = (uint8_t*)calloc(total, 1);
  uint8_t* back = (uint8_t*)calloc(total, 1);
  EXPECT(host && back);
  uint64_t seed = 7;
  for (uint64_t i = 0; i < n_bf16; ++i) {
    float f = rand_unit(&seed);
    uint32_t b;
    memcpy(&b, &f, 4);
    uint16_t h = (uint16_t)(b >> 16);
    memcpy(host + off[0] + 2 * i, &h, 2);
  }
  for (int t = 1; t < 3; ++t)
    for (uint64_t i = 0; i < bytes[t] / 4; ++i) {
      float f = rand_unit(&seed);
      memcpy(host + off[t] + 4 * i, &f, 4);
    }

  uint8_t *d_src, *d_dst;
  CHECK_CUDA(cudaMalloc((void**)&d_src, total));
  CHECK_CUDA(cudaMalloc((void**)&d_dst, total));
  CHECK_CUDA(cudaMemcpy(d_src, host, total, cudaMemcpyHostToDevice));
  CHECK_CUDA(cudaMemset(d_dst, 0x5A, total));

  fr_tensor ts[3], td[3];
  for (int t = 0; t < 3; ++t) {
    ts[t].ptr = d_src + off[t];
    td[t].ptr = d_dst + off[t];
    ts[t].nbytes = td[t].nbytes = bytes[t];
    ts[t].dtype = td[t].dtype = dtypes[t];
    ts[t].flags = td[t].flags = 0;
  }
  fr_plan ps, pd;
  CHECK_FR(fr_plan_create(ts, 3, chunk, &ps));
  CHECK_FR(fr_plan_create(td, 3, chunk, &pd));
  uint64_t C = 0, P = 0, S = 0;
  CHECK_FR(fr_plan_info(ps, &C, &P, &S));
  EXPECT(S == bytes[0] + bytes[1] + bytes[2]);
  EXPECT(C == (bytes[0] + chunk - 1) / chunk + (bytes[1] + chunk - 1) / chunk + (bytes[2] + chunk - 1) / chunk);

  uint8_t* d_packed;
  fr_fp *ta, *tb;
  uint32_t *ids, *div;
  uint64_t *cnt, *ndiv;
  CHECK_CUDA(cudaMalloc((void**)&d_packed, P));
  CHECK_CUDA(cudaMalloc((void**)&ta, C * sizeof(fr_fp)));
  CHECK_CUDA(cudaMalloc((void**)&tb, C * sizeof(fr_fp)));
  CHECK_CUDA(cudaMalloc((void**)&ids, C * 4));
  CHECK_CUDA(cudaMalloc((void**)&div, C * 4));
  CHECK_CUDA(cudaMalloc((void**)&cnt, 8));
  CHECK_CUDA(cudaMalloc((void**)&ndiv, 8));

  CHECK_FR(fr_fingerprint(ps, ta, NULL));
  CHECK_FR(fr_pack(ps, d_packed, P, NULL));
  /* damage three payloads in transit: chunks 1, C/2 and C-1 */
  const uint64_t hit[3] = {1, C / 2, C - 1};
  for (int k = 0; k < 3; ++k) {
    uint32_t ti;
    uint64_t toff, len, poff;
    CHECK_FR(fr_plan_chunk(ps, hit[k], &ti, &toff, &len, &poff));
    uint8_t v;
    CHECK_CUDA(cudaMemcpy(&v, d_packed + poff + len / 2, 1, cudaMemcpyDeviceToHost));
    v ^= 0x10;
    CHECK_CUDA(cudaMemcpy(d_packed + poff + len / 2, &v, 1, cudaMemcpyHostToDevice));
  }
  CHECK_FR(fr_unpack_verify(pd, d_packed, P, ids, C, cnt, NULL));
  uint64_t n_bad = 0;
  uint32_t bad[3] = {0, 0, 0};
  CHECK_CUDA(cudaMemcpy(&n_bad, cnt, 8, cudaMemcpyDeviceToHost));
  EXPECT(n_bad == 3);
  CHECK_CUDA(cudaMemcpy(bad, ids, 12, cudaMemcpyDeviceToHost));
  for (int k = 0; k < 3; ++k) EXPECT(bad[k] == (uint32_t)hit[k]);

  uint64_t resent = 0;
  CHECK_FR(fr_resend(ps, pd, d_packed, P, &resent, NULL, NULL));
  EXPECT(resent == 3);
  CHECK_FR(fr_unpack_collect(pd, ids, C, cnt, NULL));
  CHECK_CUDA(cudaMemcpy(&n_bad, cnt, 8, cudaMemcpyDeviceToHost));
  EXPECT(n_bad == 0);

  CHECK_FR(fr_fingerprint(pd, tb, NULL));
  CHECK_FR(fr_diff(ta, tb, C, div, C, ndiv, NULL));
  uint64_t n_div = 1;
  CHECK_CUDA(cudaMemcpy(&n_div, ndiv, 8, cudaMemcpyDeviceToHost));
  EXPECT(n_div == 0);
  CHECK_FR(fr_sync_status(pd, NULL));

  CHECK_CUDA(cudaMemcpy(back, d_dst, total, cudaMemcpyDeviceToHost));
  for (int t = 0; t < 3; ++t) EXPECT(memcmp(back + off[t], host + off[t], bytes[t]) == 0);

  fr_plan_destroy(ps);
  fr_plan_destroy(pd);
  cudaFree(d_src);
  cudaFree(d_dst);
  cudaFree(d_packed);
  cudaFree(ta);
  cudaFree(tb);
  cudaFree(ids);
  cudaFree(div);
  cudaFree(cnt);
  cudaFree(ndiv);
  free(host);
  free(back);
  printf("abi_restore ok: %llu chunks, %llu packed bytes\n", (unsigned long long)C, (unsigned long long)P);
  return 0;
}
