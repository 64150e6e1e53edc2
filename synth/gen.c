/*
 * Seeded synthetic input generator shared by the fp64 oracle and the CUDA
 * path.  It draws the inputs of the MoE-layer workloads (hidden rows, router
 * weights, expert and shared-expert weights) and holds none of the method's
 * arithmetic.
 *
 * Generator (counter-based, so any tensor of any expert can be regenerated on
 * its own and in parallel):
 *   - SplitMix64 finaliser (Steele, Lea and Flood, "Fast splittable
 *     pseudorandom number generators", OOPSLA 2014; the 64-bit mixing
 *     constants are the published ones): value i of stream `key` is
 *     mix64(key + (i + 1) * GOLDEN).
 *   - Uniforms: u = (bits >> 11) * 2^-53; the first of each pair is shifted by
 *     half an ulp so that log() never sees 0.
 *   - Normals: Box-Muller (Box and Muller 1958): pair p uses counters 2p and
 *     2p+1 and yields r*cos(theta), r*sin(theta).
 *   - Rounding: double -> float (C cast, round to nearest even) -> bf16
 *     (round to nearest even on the float bits).
 */
#include <math.h>
#include <stdint.h>

#define GOLDEN 0x9E3779B97F4A7C15ULL

static inline uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

uint64_t synth_stream_key(uint64_t seed, uint64_t tag) {
  return mix64(mix64(seed + GOLDEN) ^ mix64(tag * GOLDEN + 0x632BE59BD9B4E019ULL));
}

static inline uint16_t f32_to_bf16_rne(float f) {
  union { float f; uint32_t u; } v;
  v.f = f;
  uint32_t lsb = (v.u >> 16) & 1u;
  return (uint16_t)((v.u + 0x7FFFu + lsb) >> 16);
}

static inline void normal_pair(uint64_t key, uint64_t p, double* n0, double* n1) {
  uint64_t a = mix64(key + (2 * p + 1) * GOLDEN);
  uint64_t b = mix64(key + (2 * p + 2) * GOLDEN);
  double u1 = ((double)(a >> 11) + 0.5) * 0x1p-53;
  double u2 = (double)(b >> 11) * 0x1p-53;
  double r = sqrt(-2.0 * log(u1));
  double th = 6.283185307179586476925 * u2;
  *n0 = r * cos(th);
  *n1 = r * sin(th);
}

void synth_normal_bf16(uint64_t key, uint64_t n, double std_dev, uint16_t* out) {
  int64_t npairs = (int64_t)((n + 1) / 2);
#pragma omp parallel for schedule(static)
  for (int64_t p = 0; p < npairs; ++p) {
    double n0, n1;
    normal_pair(key, (uint64_t)p, &n0, &n1);
    out[2 * p] = f32_to_bf16_rne((float)(std_dev * n0));
    if ((uint64_t)(2 * p + 1) < n) out[2 * p + 1] = f32_to_bf16_rne((float)(std_dev * n1));
  }
}

void synth_normal_f32(uint64_t key, uint64_t n, double std_dev, float* out) {
  int64_t npairs = (int64_t)((n + 1) / 2);
#pragma omp parallel for schedule(static)
  for (int64_t p = 0; p < npairs; ++p) {
    double n0, n1;
    normal_pair(key, (uint64_t)p, &n0, &n1);
    out[2 * p] = (float)(std_dev * n0);
    if ((uint64_t)(2 * p + 1) < n) out[2 * p + 1] = (float)(std_dev * n1);
  }
}

/* Raw 64-bit stream values (used by tests of the generator itself). */
void synth_raw_u64(uint64_t key, uint64_t n, uint64_t* out) {
  for (uint64_t i = 0; i < n; ++i) out[i] = mix64(key + (i + 1) * GOLDEN);
}

/*
 * Input preparation of the 4-bit workload (not part of the method): quantise
 * bf16 weights [rows, cols] per 32 consecutive weights of a row:
 * scale = fp16(absmax / 7) (round to nearest even), q = clamp(rint(w / scale) + 8, 0, 15),
 * two codes per byte with the even column in the low nibble.
 */
static inline double bf16_to_double(uint16_t b) {
  union { uint32_t u; float f; } v;
  v.u = (uint32_t)b << 16;
  return (double)v.f;
}

void synth_quantize_q4g32(const uint16_t* w, uint64_t rows, uint64_t cols, uint8_t* packed,
                          uint16_t* scales) {
  const uint64_t groups = cols / 32;
#pragma omp parallel for schedule(static)
  for (int64_t r = 0; r < (int64_t)rows; ++r) {
    for (uint64_t g = 0; g < groups; ++g) {
      const uint16_t* src = w + (uint64_t)r * cols + g * 32;
      double amax = 0.0;
      for (int i = 0; i < 32; ++i) {
        double a = fabs(bf16_to_double(src[i]));
        if (a > amax) amax = a;
      }
      _Float16 s16 = (_Float16)(amax / 7.0);
      union { _Float16 h; uint16_t u; } sv;
      sv.h = s16;
      scales[(uint64_t)r * groups + g] = sv.u;
      const double s = (double)s16;
      uint8_t q[32];
      for (int i = 0; i < 32; ++i) {
        double v = s > 0 ? rint(bf16_to_double(src[i]) / s) + 8.0 : 8.0;
        if (v < 0) v = 0;
        if (v > 15) v = 15;
        q[i] = (uint8_t)v;
      }
      uint8_t* dst = packed + (uint64_t)r * (cols / 2) + g * 16;
      for (int i = 0; i < 16; ++i) dst[i] = (uint8_t)(q[2 * i] | (q[2 * i + 1] << 4));
    }
  }
}
