/* Host and device fill routines for the seeded synthetic inputs (see
 * synth_gen.h for the definition).  Test and benchmark infrastructure: no part
 * of the eviction method lives here.
 *
 * Layouts written (all bf16 bit patterns, row-major):
 *   keys/values of one sequence b, token positions [pos0, pos0+n):
 *       out[L][Hkv][n][D]
 *   queries of decode step `step` for sequences [0, B):
 *       out[B][L][Hq][D]
 *   new keys/values of one decode step, sequence b at position pos[b]:
 *       out[B][L][Hkv][D]
 * Regions are per token of the filled range (keys only). */
#include <cuda_runtime.h>
#include <stdint.h>
#include <string.h>

#include "synth_gen.h"

#define SYNTH_API extern "C" __attribute__((visibility("default")))

static synth_struct_params make_params(const float *kappa9) {
  synth_struct_params p;
  memset(&p, 0, sizeof(p));
  if (kappa9) {
    for (int r = 0; r < 7; ++r) p.kappa_region[r] = kappa9[r];
    p.kappa_hot = kappa9[7];
    p.kappa_q = kappa9[8];
  }
  return p;
}

/* ---------------------------------------------------------------- host ---- */

SYNTH_API uint64_t synth_key(uint64_t seed) { return synth_splitmix64(seed); }

SYNTH_API void synth_fill_kv_host(uint64_t seed, int structured, const float *kappa9,
                                  int b, int L, int Hkv, int D, int pos0, int n,
                                  const uint8_t *regions, uint16_t *k_out,
                                  uint16_t *v_out) {
  const uint64_t key = synth_splitmix64(seed);
  const synth_struct_params sp = make_params(kappa9);
  for (int l = 0; l < L; ++l)
    for (int h = 0; h < Hkv; ++h)
      for (int i = 0; i < n; ++i) {
        size_t row = (((size_t)l * Hkv + h) * n + i) * D;
        uint32_t pos = (uint32_t)(pos0 + i);
        uint32_t r = regions ? regions[i] : 0u;
        for (int d = 0; d < D; ++d) {
          if (k_out) k_out[row + d] = synth_key_bits(key, structured, &sp, b, l, h, pos, d, r);
          if (v_out) v_out[row + d] = synth_value_bits(key, b, l, h, pos, d);
        }
      }
}

SYNTH_API void synth_fill_q_host(uint64_t seed, int structured, const float *kappa9,
                                 int B, int L, int Hq, int group, int D, int step,
                                 uint16_t *q_out) {
  const uint64_t key = synth_splitmix64(seed);
  const synth_struct_params sp = make_params(kappa9);
  for (int b = 0; b < B; ++b)
    for (int l = 0; l < L; ++l)
      for (int h = 0; h < Hq; ++h) {
        size_t row = (((size_t)b * L + l) * Hq + h) * D;
        for (int d = 0; d < D; ++d)
          q_out[row + d] = synth_query_bits(key, structured, &sp, b, l, h, group, step, d);
      }
}

/* -------------------------------------------------------------- device ---- */

__global__ void synth_kv_kernel(uint64_t key, int structured, synth_struct_params sp, int b,
                                int L, int Hkv, int D, int pos0, int n,
                                const uint8_t *regions, uint16_t *k_out, uint16_t *v_out) {
  const size_t total = (size_t)L * Hkv * n * D;
  for (size_t e = (size_t)blockIdx.x * blockDim.x + threadIdx.x; e < total;
       e += (size_t)gridDim.x * blockDim.x) {
    int d = (int)(e % D);
    size_t r1 = e / D;
    int i = (int)(r1 % n);
    size_t r2 = r1 / n;
    int h = (int)(r2 % Hkv);
    int l = (int)(r2 / Hkv);
    uint32_t pos = (uint32_t)(pos0 + i);
    uint32_t reg = regions ? regions[i] : 0u;
    if (k_out) k_out[e] = synth_key_bits(key, structured, &sp, b, l, h, pos, d, reg);
    if (v_out) v_out[e] = synth_value_bits(key, b, l, h, pos, d);
  }
}

__global__ void synth_q_kernel(uint64_t key, int structured, synth_struct_params sp, int B,
                               int L, int Hq, int group, int D, int step, uint16_t *q_out) {
  const size_t total = (size_t)B * L * Hq * D;
  for (size_t e = (size_t)blockIdx.x * blockDim.x + threadIdx.x; e < total;
       e += (size_t)gridDim.x * blockDim.x) {
    int d = (int)(e % D);
    size_t r1 = e / D;
    int h = (int)(r1 % Hq);
    size_t r2 = r1 / Hq;
    int l = (int)(r2 % L);
    int b = (int)(r2 / L);
    q_out[e] = synth_query_bits(key, structured, &sp, b, l, h, group, step, d);
  }
}

/* New token of each sequence: position pos[b], region regions[b]. */
__global__ void synth_step_kv_kernel(uint64_t key, int structured, synth_struct_params sp,
                                     int B, int L, int Hkv, int D, const int32_t *pos,
                                     const uint8_t *regions, uint16_t *k_out,
                                     uint16_t *v_out) {
  const size_t total = (size_t)B * L * Hkv * D;
  for (size_t e = (size_t)blockIdx.x * blockDim.x + threadIdx.x; e < total;
       e += (size_t)gridDim.x * blockDim.x) {
    int d = (int)(e % D);
    size_t r1 = e / D;
    int h = (int)(r1 % Hkv);
    size_t r2 = r1 / Hkv;
    int l = (int)(r2 % L);
    int b = (int)(r2 / L);
    uint32_t p = (uint32_t)pos[b];
    k_out[e] = synth_key_bits(key, structured, &sp, b, l, h, p, d, regions[b]);
    v_out[e] = synth_value_bits(key, b, l, h, p, d);
  }
}

static int grid_for(size_t total) {
  size_t g = (total + 255) / 256;
  if (g > 152 * 16) g = 152 * 16;
  if (g < 1) g = 1;
  return (int)g;
}

SYNTH_API int synth_fill_kv_dev(uint64_t seed, int structured, const float *kappa9, int b,
                                int L, int Hkv, int D, int pos0, int n,
                                const uint8_t *regions_dev, void *k_dev, void *v_dev,
                                void *stream) {
  size_t total = (size_t)L * Hkv * n * D;
  if (total == 0) return 0;
  synth_kv_kernel<<<grid_for(total), 256, 0, (cudaStream_t)stream>>>(
      synth_splitmix64(seed), structured, make_params(kappa9), b, L, Hkv, D, pos0, n,
      regions_dev, (uint16_t *)k_dev, (uint16_t *)v_dev);
  return (int)cudaGetLastError();
}

SYNTH_API int synth_fill_q_dev(uint64_t seed, int structured, const float *kappa9, int B,
                               int L, int Hq, int group, int D, int step, void *q_dev,
                               void *stream) {
  size_t total = (size_t)B * L * Hq * D;
  if (total == 0) return 0;
  synth_q_kernel<<<grid_for(total), 256, 0, (cudaStream_t)stream>>>(
      synth_splitmix64(seed), structured, make_params(kappa9), B, L, Hq, group, D, step,
      (uint16_t *)q_dev);
  return (int)cudaGetLastError();
}

SYNTH_API int synth_fill_step_kv_dev(uint64_t seed, int structured, const float *kappa9,
                                     int B, int L, int Hkv, int D, const int32_t *pos_dev,
                                     const uint8_t *regions_dev, void *k_dev, void *v_dev,
                                     void *stream) {
  size_t total = (size_t)B * L * Hkv * D;
  if (total == 0) return 0;
  synth_step_kv_kernel<<<grid_for(total), 256, 0, (cudaStream_t)stream>>>(
      synth_splitmix64(seed), structured, make_params(kappa9), B, L, Hkv, D, pos_dev,
      regions_dev, (uint16_t *)k_dev, (uint16_t *)v_dev);
  return (int)cudaGetLastError();
}
