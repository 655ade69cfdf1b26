/*
 * Seeded synthetic input generator shared by the CUDA path's tests/bench and
 * the CPU oracle's tests.  It holds none of the attention or compaction
 * arithmetic: it only maps an element's coordinates to a 16-bit float.
 *
 * Generator: Philox4x32-10, the counter-based generator published by
 * Salmon, Moraes, Dror and Shaw ("Parallel Random Numbers: As Easy as 1, 2, 3",
 * SC 2011): 10 rounds of two 32x32->64 multiplies with the published
 * multipliers and Weyl key increments.
 *
 * Element value: the four output words give four 16-bit uniforms (their high
 * halves); their sum S lies in [0, 262140] and has mean 131070 and standard
 * deviation 65536/sqrt(3).  x = float(S - 131070) * scale is computed as ONE
 * IEEE binary32 multiply (round to nearest even), then rounded once more, to
 * nearest even, to binary16 or bfloat16.  With scale = sigma*sqrt(3)/65536
 * the values approximate N(0, sigma^2) (Irwin-Hall of order 4) with tails cut
 * at about 3.46 sigma.  Every step is exact or correctly rounded, so the host
 * and device builds of this header give identical bits.
 *
 * Counter layout: ctr = {i0, i1, i2, tag}, key = {seed_lo, seed_hi}.  The
 * callers use i0 = token index, i1 = sequence, i2 = head*1024 + dim and
 * tag = tensor (0 K, 1 V, 2 q) | layer << 8.
 */
#ifndef SYNTH_GEN_H
#define SYNTH_GEN_H

#include <stdint.h>

#if defined(__CUDACC__)
#define SYN_FN static __host__ __device__ __forceinline__
#else
#define SYN_FN static inline
#endif

#define SYN_DTYPE_F16 0
#define SYN_DTYPE_BF16 1

SYN_FN void syn_mulhilo(uint32_t a, uint32_t b, uint32_t* hi, uint32_t* lo) {
  uint64_t p = (uint64_t)a * (uint64_t)b;
  *hi = (uint32_t)(p >> 32);
  *lo = (uint32_t)p;
}

/* Philox4x32 with 10 rounds. */
SYN_FN void syn_philox4x32_10(const uint32_t in[4], uint32_t k0, uint32_t k1, uint32_t out[4]) {
  uint32_t c0 = in[0], c1 = in[1], c2 = in[2], c3 = in[3];
  for (int r = 0; r < 10; ++r) {
    uint32_t hi0, lo0, hi1, lo1;
    syn_mulhilo(0xD2511F53u, c0, &hi0, &lo0);
    syn_mulhilo(0xCD9E8D57u, c2, &hi1, &lo1);
    uint32_t n0 = hi1 ^ c1 ^ k0;
    uint32_t n2 = hi0 ^ c3 ^ k1;
    c0 = n0;
    c1 = lo1;
    c2 = n2;
    c3 = lo0;
    k0 += 0x9E3779B9u;
    k1 += 0xBB67AE85u;
  }
  out[0] = c0;
  out[1] = c1;
  out[2] = c2;
  out[3] = c3;
}

/* Centred Irwin-Hall(4) integer in [-131070, 131070]. */
SYN_FN int32_t syn_centred_sum(uint64_t seed, uint32_t tag, uint32_t i0, uint32_t i1, uint32_t i2) {
  uint32_t ctr[4] = {i0, i1, i2, tag};
  uint32_t w[4];
  syn_philox4x32_10(ctr, (uint32_t)seed, (uint32_t)(seed >> 32), w);
  int32_t s = (int32_t)(w[0] >> 16) + (int32_t)(w[1] >> 16) + (int32_t)(w[2] >> 16) + (int32_t)(w[3] >> 16);
  return s - 131070;
}

#endif
