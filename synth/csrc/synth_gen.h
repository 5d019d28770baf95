/* Seeded synthetic-input generator shared by the fp64 oracle's test harness and
 * the GPU benchmark.  It holds none of the eviction method's arithmetic: it only
 * turns (seed, tensor, indices) into bf16 bit patterns, the same on the host and
 * on the device.
 *
 * Definition (bit-exact on every side that implements it):
 *   key   = splitmix64(seed)
 *   ctr   = tensor<<60 | b<<48 | l<<40 | h<<34 | pos<<8 | d
 *   z     = splitmix64(ctr ^ key)
 *   S     = sum of the four 16-bit fields of z          (Irwin-Hall, n = 4)
 *   v     = (float)(S - 131070) * SYNTH_NORM            (one fp32 multiply, RN)
 *   value = bf16 round-to-nearest-even of v
 * splitmix64 is the finaliser published by Steele, Lea and Flood (OOPSLA 2014,
 * "Fast splittable pseudorandom number generators"), as used in Vigna's
 * xoshiro seeding.  S has mean 131070 and standard deviation
 * sqrt((65536^2-1)/3) = 37837.23, so v is close to N(0,1).
 *
 * "Structured" keys/queries add a per-(layer, kv-head) sign pattern on the
 * first SYNTH_STRUCT_DIMS dimensions, scaled per region, so that regions draw
 * different attention mass (a logit offset of kappa_q*kappa_r*16/sqrt(128)), and
 * a seeded ~2% of tokens get an extra "hot" offset.  The add is one fp32 add
 * of exactly representable values before the bf16 rounding.
 */
#ifndef MD_SYNTH_GEN_H
#define MD_SYNTH_GEN_H

#include <stdint.h>

#if defined(__CUDACC__)
#define SYNTH_HD __host__ __device__ __forceinline__
#else
#define SYNTH_HD static inline
#endif

enum {
  SYNTH_T_K = 1,      /* keys,    index (b, l, kv head, token position, d)   */
  SYNTH_T_V = 2,      /* values,  index (b, l, kv head, token position, d)   */
  SYNTH_T_Q = 3,      /* queries, index (b, l, q head, decode step, d)       */
  SYNTH_T_SIGN = 5,   /* structure sign pattern, index (0, l, kv head, 0, d) */
  SYNTH_T_HOT = 6     /* hot-token draw, index (b, 0, 0, token position, 0)  */
};

#define SYNTH_NORM 2.6429130e-05f /* 1/37837.23, rounded to fp32 */
#define SYNTH_STRUCT_DIMS 16
/* 2% of 2^24: a token is "hot" when the top 24 bits of its draw fall below. */
#define SYNTH_HOT_THRESHOLD 335544u

SYNTH_HD uint64_t synth_splitmix64(uint64_t x) {
  uint64_t z = x + 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

SYNTH_HD uint64_t synth_ctr(uint32_t tensor, uint32_t b, uint32_t l, uint32_t h,
                            uint32_t pos, uint32_t d) {
  return ((uint64_t)(tensor & 0xFu) << 60) | ((uint64_t)(b & 0xFFFu) << 48) |
         ((uint64_t)(l & 0xFFu) << 40) | ((uint64_t)(h & 0x3Fu) << 34) |
         ((uint64_t)(pos & 0x3FFFFFFu) << 8) | (uint64_t)(d & 0xFFu);
}

SYNTH_HD uint32_t synth_f32_bits(float f) {
  union { float f; uint32_t u; } c;
  c.f = f;
  return c.u;
}

SYNTH_HD float synth_bits_f32(uint32_t u) {
  union { float f; uint32_t u; } c;
  c.u = u;
  return c.f;
}

/* fp32 -> bf16 bits, round to nearest, ties to even (inputs are finite). */
SYNTH_HD uint16_t synth_bf16_rne(float f) {
  uint32_t u = synth_f32_bits(f);
  u += 0x7FFFu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

/* The fp32 value before bf16 rounding, ~N(0,1). */
SYNTH_HD float synth_normal_f32(uint64_t key, uint32_t tensor, uint32_t b, uint32_t l,
                                uint32_t h, uint32_t pos, uint32_t d) {
  uint64_t z = synth_splitmix64(synth_ctr(tensor, b, l, h, pos, d) ^ key);
  int32_t s = (int32_t)(z & 0xFFFFu) + (int32_t)((z >> 16) & 0xFFFFu) +
              (int32_t)((z >> 32) & 0xFFFFu) + (int32_t)((z >> 48) & 0xFFFFu);
  float v = (float)(s - 131070);
#if defined(__CUDA_ARCH__)
  return __fmul_rn(v, SYNTH_NORM);
#else
  return v * SYNTH_NORM;
#endif
}

SYNTH_HD float synth_sign(uint64_t key, uint32_t l, uint32_t kvh, uint32_t d) {
  uint64_t z = synth_splitmix64(synth_ctr(SYNTH_T_SIGN, 0, l, kvh, 0, d) ^ key);
  return (z & 1u) ? 1.0f : -1.0f;
}

SYNTH_HD int synth_is_hot(uint64_t key, uint32_t b, uint32_t pos) {
  uint64_t z = synth_splitmix64(synth_ctr(SYNTH_T_HOT, b, 0, 0, pos, 0) ^ key);
  return (uint32_t)(z >> 40) < SYNTH_HOT_THRESHOLD;
}

SYNTH_HD float synth_add_rn(float a, float b) {
#if defined(__CUDA_ARCH__)
  return __fadd_rn(a, b);
#else
  return a + b;
#endif
}

/* Structure offsets.  kappa[r] for keys of region r (7 regions), then kappa_hot
 * for hot keys and kappa_q for queries; all multiples of 1/64 (exact). */
typedef struct {
  float kappa_region[8];
  float kappa_hot;
  float kappa_q;
} synth_struct_params;

/* Key element (b, l, kvh, pos, d) as bf16 bits. */
SYNTH_HD uint16_t synth_key_bits(uint64_t key, int structured, const synth_struct_params *sp,
                                 uint32_t b, uint32_t l, uint32_t kvh, uint32_t pos,
                                 uint32_t d, uint32_t region) {
  float v = synth_normal_f32(key, SYNTH_T_K, b, l, kvh, pos, d);
  if (structured && d < SYNTH_STRUCT_DIMS) {
    float k = sp->kappa_region[region & 7u];
    if (synth_is_hot(key, b, pos)) k = synth_add_rn(k, sp->kappa_hot);
    v = synth_add_rn(v, k * synth_sign(key, l, kvh, d));
  }
  return synth_bf16_rne(v);
}

SYNTH_HD uint16_t synth_value_bits(uint64_t key, uint32_t b, uint32_t l, uint32_t kvh,
                                   uint32_t pos, uint32_t d) {
  return synth_bf16_rne(synth_normal_f32(key, SYNTH_T_V, b, l, kvh, pos, d));
}

/* Query element (b, l, q head hq, decode step, d); group = q heads per kv head. */
SYNTH_HD uint16_t synth_query_bits(uint64_t key, int structured, const synth_struct_params *sp,
                                   uint32_t b, uint32_t l, uint32_t hq, uint32_t group,
                                   uint32_t step, uint32_t d) {
  float v = synth_normal_f32(key, SYNTH_T_Q, b, l, hq, step, d);
  if (structured && d < SYNTH_STRUCT_DIMS)
    v = synth_add_rn(v, sp->kappa_q * synth_sign(key, l, hq / group, d));
  return synth_bf16_rne(v);
}

#endif /* MD_SYNTH_GEN_H */
