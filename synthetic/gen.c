/*
 * Seeded synthetic inputs for the PARD decode-step workloads.
 *
 * This file holds no arithmetic of the method itself: it only turns a seed
 * into weights, prompt ids, prompt lengths and page orders.  Both the CPU
 * oracle and the CUDA path consume its output, so neither has to trust the
 * other for inputs.
 *
 * Generator: SplitMix64 (Steele, Lea, Flood, "Fast splittable pseudorandom
 * number generators", OOPSLA 2014) used as a counter-based hash: the value
 * for element i of stream s is mix64(s * GOLDEN + i), where mix64 is the
 * SplitMix64 output finaliser.  Normal samples come from the Box-Muller
 * transform in double precision and are rounded to bf16 with
 * round-to-nearest-even, so the stored bits are what every consumer sees.
 *
 * Host-only, portable C99 (no intrinsics); identical results on x86-64 and
 * aarch64 up to the last bit of libm's double log/sin/cos, which bf16
 * rounding hides in all but ~2^-40 of the elements.
 */
#include <math.h>
#include <stddef.h>
#include <stdint.h>

#define GOLDEN 0x9E3779B97F4A7C15ULL

static inline uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

/* stream id from (seed, tag): distinct tags give unrelated streams */
static inline uint64_t stream_of(uint64_t seed, uint64_t tag) {
  return mix64(seed * GOLDEN + mix64(tag + 0x632BE59BD9B4E019ULL));
}

static inline uint64_t draw(uint64_t stream, uint64_t i) {
  return mix64(stream + (i + 1) * GOLDEN);
}

static inline uint16_t f32_to_bf16_rne(float f) {
  union { float f; uint32_t u; } v;
  v.f = f;
  uint32_t u = v.u;
  if ((u & 0x7F800000u) == 0x7F800000u && (u & 0x007FFFFFu)) return (uint16_t)((u >> 16) | 0x40);
  u += 0x7FFFu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

/* n bf16 values ~ N(0, std^2).  Pair j uses draws 2j (u1 in (0,1]) and
 * 2j+1 (u2 in [0,1)); element 2j gets the cosine branch, 2j+1 the sine. */
void synth_normal_bf16(uint64_t seed, uint64_t tag, double std, uint16_t* out, int64_t n) {
  const uint64_t s = stream_of(seed, tag);
  const double two_pi = 6.283185307179586476925286766559;
  const int64_t npairs = (n + 1) / 2;
#pragma omp parallel for schedule(static)
  for (int64_t j = 0; j < npairs; ++j) {
    uint64_t a = draw(s, 2 * (uint64_t)j), b = draw(s, 2 * (uint64_t)j + 1);
    double u1 = ((double)(a >> 11) + 1.0) * (1.0 / 9007199254740992.0); /* (0,1] */
    double u2 = (double)(b >> 11) * (1.0 / 9007199254740992.0);         /* [0,1) */
    double r = sqrt(-2.0 * log(u1));
    double z0 = r * cos(two_pi * u2), z1 = r * sin(two_pi * u2);
    out[2 * j] = f32_to_bf16_rne((float)(std * z0));
    if (2 * j + 1 < n) out[2 * j + 1] = f32_to_bf16_rne((float)(std * z1));
  }
}

void synth_fill_bf16(uint16_t bits, uint16_t* out, int64_t n) {
#pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < n; ++i) out[i] = bits;
}

/* n integers uniform in [lo, lo + span) (span >= 1), modulo reduction of a
 * 64-bit draw (bias below 2^-40 for the spans used here). */
void synth_uniform_int(uint64_t seed, uint64_t tag, int64_t lo, int64_t span, int32_t* out, int64_t n) {
  const uint64_t s = stream_of(seed, tag);
  for (int64_t i = 0; i < n; ++i) out[i] = (int32_t)(lo + (int64_t)(draw(s, (uint64_t)i) % (uint64_t)span));
}

/* Fisher-Yates permutation of 0..n-1 driven by the same stream. */
void synth_permutation(uint64_t seed, uint64_t tag, int32_t* out, int64_t n) {
  const uint64_t s = stream_of(seed, tag);
  for (int64_t i = 0; i < n; ++i) out[i] = (int32_t)i;
  for (int64_t i = n - 1; i > 0; --i) {
    int64_t j = (int64_t)(draw(s, (uint64_t)i) % (uint64_t)(i + 1));
    int32_t t = out[i]; out[i] = out[j]; out[j] = t;
  }
}
