/*
 * Host build of the seeded synthetic input generator (see synth_gen.h for the
 * definition).  Used by the tests and the CPU baseline to regenerate any slice
 * of a workload's K, V and q without copying it back from the GPU.
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

#include "synth_gen.h"

/* binary32 -> binary16, round to nearest, ties to even (IEEE 754-2008 4.3.1). */
uint16_t syn_f32_to_f16(float f) {
  uint32_t x;
  memcpy(&x, &f, 4);
  uint32_t sign = (x >> 16) & 0x8000u;
  uint32_t ax = x & 0x7FFFFFFFu;
  if (ax > 0x7F800000u) return (uint16_t)(sign | 0x7E00u); /* NaN */
  if (ax >= 0x477FF000u) return (uint16_t)(sign | 0x7C00u); /* >= 65520: overflows to inf */
  if (ax < 0x00800000u) return (uint16_t)sign;              /* binary32 subnormal: far below 2^-25 */
  int e = (int)(ax >> 23) - 127;
  uint32_t m = (ax & 0x7FFFFFu) | 0x800000u; /* 24-bit significand */
  if (e >= -14) {
    /* normal binary16: keep 11 significant bits */
    uint32_t r = ((uint32_t)(e + 15) << 10) | ((m >> 13) & 0x3FFu);
    uint32_t rem = m & 0x1FFFu;
    if (rem > 0x1000u || (rem == 0x1000u && (r & 1u))) r += 1u;
    return (uint16_t)(sign | r);
  }
  /* subnormal binary16: value = m * 2^(e-23); unit 2^-24 -> m * 2^(e+1) */
  int s = -1 - e; /* right shift, >= 14 */
  if (s > 24) return (uint16_t)sign;
  uint32_t r = m >> s;
  uint32_t rem = m & ((1u << s) - 1u);
  uint32_t half = 1u << (s - 1);
  if (rem > half || (rem == half && (r & 1u))) r += 1u;
  return (uint16_t)(sign | r);
}

/* binary32 -> bfloat16, round to nearest, ties to even. */
uint16_t syn_f32_to_bf16(float f) {
  uint32_t x;
  memcpy(&x, &f, 4);
  if ((x & 0x7FFFFFFFu) > 0x7F800000u) return (uint16_t)(((x >> 16) & 0x8000u) | 0x7FC0u);
  uint32_t lsb = (x >> 16) & 1u;
  return (uint16_t)((x + 0x7FFFu + lsb) >> 16);
}

/* One element: the IEEE binary32 product, then one rounding to the 16-bit type. */
uint16_t syn_value(uint64_t seed, int dtype, float scale, uint32_t tag, uint32_t i0, uint32_t i1, uint32_t i2) {
  float c = (float)syn_centred_sum(seed, tag, i0, i1, i2); /* exact: |c| < 2^24 */
  float x = c * scale;                                     /* one binary32 rounding (built with -ffp-contract=off) */
  return dtype == SYN_DTYPE_BF16 ? syn_f32_to_bf16(x) : syn_f32_to_f16(x);
}

/*
 * out[(tok*H + h)*d + e] = value(tag, i0 = tok_t[tok], i1 = tok_s[tok], i2 = h*1024 + e)
 * Layout [n_tok][H][d], the same as the device fill.
 */
void syn_fill_tokens(uint64_t seed, int dtype, float scale, uint32_t tag, int64_t n_tok, const int32_t* tok_t,
                     const int32_t* tok_s, int H, int d, uint16_t* out) {
#pragma omp parallel for schedule(static)
  for (int64_t tok = 0; tok < n_tok; ++tok) {
    for (int h = 0; h < H; ++h) {
      for (int e = 0; e < d; ++e) {
        out[(tok * H + h) * d + e] = syn_value(seed, dtype, scale, tag, (uint32_t)tok_t[tok], (uint32_t)tok_s[tok],
                                               (uint32_t)(h * 1024 + e));
      }
    }
  }
}

/* Raw centred sums (for statistical tests of the generator). */
void syn_centred_sums(uint64_t seed, uint32_t tag, int64_t n, const uint32_t* i0, const uint32_t* i1,
                      const uint32_t* i2, int32_t* out) {
#pragma omp parallel for schedule(static)
  for (int64_t k = 0; k < n; ++k) out[k] = syn_centred_sum(seed, tag, i0[k], i1[k], i2[k]);
}

/* Raw Philox4x32-10 blocks. */
void syn_philox_blocks(int64_t n, const uint32_t* ctr4, const uint32_t* key2, uint32_t* out4) {
  for (int64_t k = 0; k < n; ++k) syn_philox4x32_10(ctr4 + 4 * k, key2[2 * k], key2[2 * k + 1], out4 + 4 * k);
}

/* Vector conversions, exposed so tests can compare them with library routines. */
void syn_f32_to_f16_array(int64_t n, const float* in, uint16_t* out) {
  for (int64_t k = 0; k < n; ++k) out[k] = syn_f32_to_f16(in[k]);
}
void syn_f32_to_bf16_array(int64_t n, const float* in, uint16_t* out) {
  for (int64_t k = 0; k < n; ++k) out[k] = syn_f32_to_bf16(in[k]);
}
