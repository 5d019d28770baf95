/* A plain C caller of the library: the boundary without Python.  One small
 * cache (1 layer, 8/2 heads, pages of 16), a 300-token trace in two regions,
 * four decode steps through md_decode_step_host, then an eviction to a budget
 * of 10 pages.  Checks the statuses, that the outputs are finite, and that the
 * sequence ends within its budget.  Prints "ok" and exits 0 on success. */
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <cuda_runtime_api.h>

#include "memdecay.h"

#define CHECK(x)                                                              \
  do {                                                                        \
    int s_ = (int)(x);                                                        \
    if (s_ < 0) {                                                             \
      fprintf(stderr, "%s failed: %d\n", #x, s_);                             \
      return 1;                                                               \
    }                                                                         \
  } while (0)

/* bf16 bits of a float (round to nearest even; inputs are finite) */
static uint16_t bf16(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  u += 0x7FFFu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

static float f32(uint16_t h) {
  uint32_t u = (uint32_t)h << 16;
  float f;
  memcpy(&f, &u, 4);
  return f;
}

static uint32_t lcg(uint32_t *s) {
  *s = *s * 1664525u + 1013904223u;
  return *s >> 8;
}

int main(void) {
  const int L = 1, Hq = 8, Hkv = 2, D = 128, ps = 16, n0 = 300, steps = 4, budget = 10;
  md_config cfg;
  memset(&cfg, 0, sizeof(cfg));
  cfg.num_layers = L;
  cfg.num_q_heads = Hq;
  cfg.num_kv_heads = Hkv;
  cfg.head_dim = D;
  cfg.page_size = ps;
  cfg.max_batch = 1;
  cfg.max_pages_per_seq = 64;
  cfg.num_phys_pages = 64;
  cfg.rho = 0.9f;
  cfg.gamma = 0.1f;
  cfg.tau_scale = 2.0f;
  cfg.attn_weight = 1.0f;
  cfg.keep_token_prio = 1;
  const size_t ws = md_workspace_size(&cfg);
  if (ws == 0) {
    fprintf(stderr, "configuration rejected\n");
    return 1;
  }
  if (cudaMalloc(&cfg.workspace, ws) != cudaSuccess) return 1;
  cfg.workspace_bytes = ws;
  md_ctx *ctx = NULL;
  CHECK(md_create(&cfg, &ctx));
  for (int r = 0; r < MD_NUM_REGIONS; ++r)
    CHECK(md_set_region_params(ctx, r, 1.0f - 0.1f * (float)r, 20.0f + 10.0f * (float)r, r == MD_REGION_SYSTEM));

  /* the trace: 40 pinned system tokens, then user tokens; K/V [L][Hkv][n][D] */
  uint32_t seed = 7u;
  uint8_t *regions = malloc(n0);
  uint16_t *k = malloc((size_t)L * Hkv * n0 * D * 2), *v = malloc((size_t)L * Hkv * n0 * D * 2);
  for (int i = 0; i < n0; ++i) regions[i] = i < 40 ? MD_REGION_SYSTEM : MD_REGION_USER;
  for (size_t i = 0; i < (size_t)L * Hkv * n0 * D; ++i) {
    k[i] = bf16(((float)(lcg(&seed) % 2001) - 1000.0f) / 1000.0f);
    v[i] = bf16(((float)(lcg(&seed) % 2001) - 1000.0f) / 1000.0f);
  }
  void *kd = NULL, *vd = NULL;
  if (cudaMalloc(&kd, (size_t)L * Hkv * n0 * D * 2) != cudaSuccess ||
      cudaMalloc(&vd, (size_t)L * Hkv * n0 * D * 2) != cudaSuccess)
    return 1;
  cudaMemcpy(kd, k, (size_t)L * Hkv * n0 * D * 2, cudaMemcpyHostToDevice);
  cudaMemcpy(vd, v, (size_t)L * Hkv * n0 * D * 2, cudaMemcpyHostToDevice);
  CHECK(md_append_tokens(ctx, 0, n0, regions, NULL, kd, vd));

  uint16_t q[1 * 1 * 8 * 128], kn[1 * 1 * 2 * 128], vn[1 * 1 * 2 * 128], out[1 * 1 * 8 * 128];
  const uint8_t reg_new = MD_REGION_SCRATCHPAD;
  for (int t = 0; t < steps; ++t) {
    for (int i = 0; i < Hq * D; ++i) q[i] = bf16(((float)(lcg(&seed) % 2001) - 1000.0f) / 1000.0f);
    for (int i = 0; i < Hkv * D; ++i) {
      kn[i] = bf16(((float)(lcg(&seed) % 2001) - 1000.0f) / 1000.0f);
      vn[i] = bf16(((float)(lcg(&seed) % 2001) - 1000.0f) / 1000.0f);
    }
    CHECK(md_decode_step_host(ctx, 1, q, kn, vn, &reg_new, out));
    CHECK(md_sync(ctx));
    for (int i = 0; i < Hq * D; ++i)
      if (!isfinite(f32(out[i]))) {
        fprintf(stderr, "non-finite output\n");
        return 1;
      }
    const int32_t bud = budget;
    int32_t n_ev = -1;
    CHECK(md_evict(ctx, 1, &bud, &n_ev, NULL));
  }
  CHECK(md_sync(ctx));
  int64_t pages = -1;
  CHECK(md_query(ctx, MD_QUERY_PAGES, 0, &pages));
  if (pages > budget) {
    fprintf(stderr, "%lld pages after eviction, budget %d\n", (long long)pages, budget);
    return 1;
  }
  CHECK(md_destroy(ctx));
  cudaFree(kd);
  cudaFree(vd);
  cudaFree(cfg.workspace);
  free(regions);
  free(k);
  free(v);
  printf("ok\n");
  return 0;
}
