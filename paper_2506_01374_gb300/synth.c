/* Fast path of the seeded input generator (inputs.py): N(mean, std^2)
 * samples stored as bf16 bit patterns. Same definition as the numpy path:
 * element i of stream `key` uses splitmix64 draws 2i and 2i+1,
 *   d_n = mix(key + (n + 1) * 0x9E3779B97F4A7C15),  u = (d >> 11) * 2^-53,
 *   z = mean + std * sqrt(-2 ln(1 - u1)) * cos(2 pi u2),
 * rounded to fp32, then to bf16 with round-to-nearest-even. Holds no
 * operator arithmetic; it only draws inputs. */
#include <math.h>
#include <stdint.h>
#include <string.h>

static inline uint64_t mix(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

__attribute__((visibility("default"))) void synth_bf16_normal(uint64_t key, int64_t start, int64_t n, double mean,
                                                              double std, uint16_t* out) {
  const uint64_t G = 0x9E3779B97F4A7C15ull;
  const double two_pi = 6.283185307179586476925286766559;
#pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < n; ++i) {
    const uint64_t c = (uint64_t)(start + i);
    const uint64_t d1 = mix(key + (2 * c + 1) * G);
    const uint64_t d2 = mix(key + (2 * c + 2) * G);
    const double u1 = (double)(d1 >> 11) * 0x1p-53;
    const double u2 = (double)(d2 >> 11) * 0x1p-53;
    const double z = mean + std * sqrt(-2.0 * log1p(-u1)) * cos(two_pi * u2);
    float f = (float)z;
    uint32_t u;
    memcpy(&u, &f, 4);
    u = (u + 0x7FFFu + ((u >> 16) & 1u)) >> 16;
    out[i] = (uint16_t)u;
  }
}
