/* Multi-threaded host implementation of the seeded input generator.
 *
 * Same definition as the numpy generator in synth.py (splitmix64 finaliser
 * of Steele, Lea and Flood, OOPSLA 2014, as a counter-based stream; uniforms
 * ((w >> 11) + 0.5) * 2^-53; Box-Muller normals on consecutive pairs; value
 * scaled in double, rounded to float and then to bf16, both round to nearest
 * even).  It only draws random numbers: no LoRA arithmetic lives here.
 * Built with -ffp-contract=off so that no multiply-add is fused and each
 * double operation rounds exactly as numpy's does.
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

static const uint64_t G = 0x9E3779B97F4A7C15ull;

static inline uint64_t mix64(uint64_t z) {
  z ^= z >> 30; z *= 0xBF58476D1CE4E5B9ull;
  z ^= z >> 27; z *= 0x94D049BB133111EBull;
  z ^= z >> 31;
  return z;
}

static inline double u01(uint64_t key, uint64_t i) { /* element i (0-based) */
  uint64_t w = mix64(key + (i + 1) * G);
  return ((double)(w >> 11) + 0.5) * 0x1p-53;
}

static inline uint16_t bf16_rne(double v) {
  float f = (float)v;
  uint32_t u; memcpy(&u, &f, 4);
  u = (u + 0x7FFFu + ((u >> 16) & 1u)) >> 16;
  return (uint16_t)u;
}

void synth_normal_bf16(uint64_t key, int64_t n, double std_, uint16_t* out) {
  const int64_t m = (n + 1) / 2;
  const double two_pi = 6.283185307179586; /* double nearest to 2*pi, as math.pi*2.0 */
  #pragma omp parallel for schedule(static)
  for (int64_t p = 0; p < m; ++p) {
    double a = u01(key, (uint64_t)(2 * p));
    double b = u01(key, (uint64_t)(2 * p + 1));
    double rho = sqrt(-2.0 * log(a));
    double ang = two_pi * b;
    double z0 = rho * cos(ang), z1 = rho * sin(ang);
    out[2 * p] = bf16_rne(z0 * std_);
    if (2 * p + 1 < n) out[2 * p + 1] = bf16_rne(z1 * std_);
  }
}

void synth_uniform_bf16(uint64_t key, int64_t n, double bound, uint16_t* out) {
  #pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < n; ++i) {
    double u = u01(key, (uint64_t)i);
    out[i] = bf16_rne((2.0 * u - 1.0) * bound);
  }
}
