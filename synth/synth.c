/*
 * Seeded synthetic inputs for the capped-residency MoE decode step.
 *
 * This module generates workload data only: weights, hidden-state streams, and
 * their storage encodings (bf16 rounding, symmetric int4 g128 quantisation).
 * It contains none of the decode step's arithmetic (no routing, no residency,
 * no expert FFN) and is shared by the fp64 oracle and by the CUDA path as the
 * single source of input values.
 *
 * Random numbers are counter-based so that any (seed, stream, index) is
 * reproducible independently of generation order and thread count:
 *   - the integer hash is the SplitMix64 output function (Steele, Lea & Flood,
 *     "Fast Splittable Pseudorandom Number Generators", OOPSLA 2014), applied
 *     to key + (counter + 1) * golden-gamma;
 *   - normals come from the Box-Muller transform (Box & Muller, 1958) of two
 *     24-bit uniforms taken from one 64-bit hash.
 *
 * Built with -ffp-contract=off so that no multiply-add is fused differently on
 * x86_64 and aarch64.
 */
#define _GNU_SOURCE
#include <math.h>
#include <stdint.h>
#include <string.h>

#define SYNTH_GAMMA 0x9E3779B97F4A7C15ULL

static inline uint64_t sm64_mix(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

/* Key of one random stream: a SplitMix64 state derived from (seed, stream). */
uint64_t synth_key(uint64_t seed, uint64_t stream) {
  return sm64_mix(sm64_mix(seed * SYNTH_GAMMA + 0x1234567ULL) ^ (stream + SYNTH_GAMMA));
}

/* Raw 64-bit hash number `counter` of the stream with the given key. */
uint64_t synth_hash(uint64_t key, uint64_t counter) {
  return sm64_mix(key + (counter + 1ULL) * SYNTH_GAMMA);
}

static inline void box_muller_pair(uint64_t x, float* z0, float* z1) {
  /* u1 in (0, 1], u2 in [0, 1), 24 bits each. */
  const float inv24 = 1.0f / 16777216.0f;
  float u1 = (float)((x >> 40) + 1ULL) * inv24;
  float u2 = (float)((x >> 16) & 0xFFFFFFULL) * inv24;
  float r = sqrtf(-2.0f * logf(u1));
  float th = 6.2831853071795864769f * u2;
  float sn, cs;
  sincosf(th, &sn, &cs);
  *z0 = r * cs;
  *z1 = r * sn;
}

/* out[i] = std * N(0,1) number (start + i) of stream (seed, stream). Normal number
 * 2p is the cosine branch and 2p+1 the sine branch of Box-Muller pair p. */
void synth_normal(uint64_t seed, uint64_t stream, uint64_t start, int64_t n, float std, float* out) {
  uint64_t key = synth_key(seed, stream);
  int64_t i = 0;
  uint64_t j = start;
  float z0, z1;
  if (n <= 0) return;
  if (j & 1ULL) {
    box_muller_pair(synth_hash(key, j >> 1), &z0, &z1);
    out[i++] = std * z1;
    j++;
  }
  for (; i + 1 < n; i += 2, j += 2) {
    box_muller_pair(synth_hash(key, j >> 1), &z0, &z1);
    out[i] = std * z0;
    out[i + 1] = std * z1;
  }
  if (i < n) {
    box_muller_pair(synth_hash(key, j >> 1), &z0, &z1);
    out[i] = std * z0;
  }
}

/* float -> bf16 bits, round to nearest even; NaN stays a quiet NaN. */
static inline uint16_t f32_to_bf16(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  if ((u & 0x7F800000u) == 0x7F800000u && (u & 0x007FFFFFu)) return (uint16_t)((u >> 16) | 0x0040u);
  uint32_t lsb = (u >> 16) & 1u;
  u += 0x7FFFu + lsb;
  return (uint16_t)(u >> 16);
}

static inline float bf16_to_f32(uint16_t b) {
  uint32_t u = (uint32_t)b << 16;
  float f;
  memcpy(&f, &u, 4);
  return f;
}

void synth_f32_to_bf16(const float* in, uint16_t* out, int64_t n) {
  for (int64_t i = 0; i < n; i++) out[i] = f32_to_bf16(in[i]);
}

void synth_f64_to_f32(const double* in, float* out, int64_t n) {
  for (int64_t i = 0; i < n; i++) out[i] = (float)in[i];
}

/* f64 -> f32 (round to nearest) -> bf16 (round to nearest even). */
void synth_f64_to_bf16(const double* in, uint16_t* out, int64_t n) {
  for (int64_t i = 0; i < n; i++) out[i] = f32_to_bf16((float)in[i]);
}

/*
 * AR(1) hidden stream, T states of dimension d, in fp64:
 *   h_0 = eps_0,  h_t = rho * h_{t-1} + sqrt(1 - rho^2) * eps_t,
 * eps_t[i] = normal number (t*d + i) of stream (seed, stream). Unit stationary
 * variance. `scratch` holds d floats.
 */
void synth_ar1(uint64_t seed, uint64_t stream, int64_t T, int64_t d, double rho, double* out, float* scratch) {
  double c = sqrt(1.0 - rho * rho);
  for (int64_t t = 0; t < T; t++) {
    synth_normal(seed, stream, (uint64_t)(t * d), d, 1.0f, scratch);
    double* h = out + t * d;
    if (t == 0) {
      for (int64_t i = 0; i < d; i++) h[i] = (double)scratch[i];
    } else {
      const double* hp = h - d;
      for (int64_t i = 0; i < d; i++) h[i] = rho * hp[i] + c * (double)scratch[i];
    }
  }
}

/*
 * Symmetric int4 quantisation, groups of 128 consecutive elements along each
 * row (the input dimension), bf16 scales:
 *   scale = bf16(absmax / 7);  q = clamp(rint_even(w / scale), -7, 7)  (q = 0 if scale == 0).
 * Packing: byte j of a row holds element 2j in its low nibble and 2j+1 in its
 * high nibble, two's complement. cols must be a multiple of 128.
 * q has rows*cols/2 bytes, scales rows*cols/128 entries.
 */
int synth_quant_int4_g128(const float* w, int64_t rows, int64_t cols, uint8_t* q, uint16_t* scales) {
  if (cols % 128 != 0) return -1;
  int64_t groups = cols / 128;
  for (int64_t r = 0; r < rows; r++) {
    for (int64_t g = 0; g < groups; g++) {
      const float* src = w + r * cols + g * 128;
      float amax = 0.0f;
      for (int i = 0; i < 128; i++) {
        float a = fabsf(src[i]);
        if (a > amax) amax = a;
      }
      uint16_t sb = f32_to_bf16(amax / 7.0f);
      float s = bf16_to_f32(sb);
      scales[r * groups + g] = sb;
      uint8_t* dst = q + (r * cols + g * 128) / 2;
      for (int i = 0; i < 128; i += 2) {
        int v[2];
        for (int h = 0; h < 2; h++) {
          int qi = 0;
          if (s != 0.0f) {
            float t = nearbyintf(src[i + h] / s);
            if (t > 7.0f) t = 7.0f;
            if (t < -7.0f) t = -7.0f;
            qi = (int)t;
          }
          v[h] = qi;
        }
        dst[i / 2] = (uint8_t)(((unsigned)v[0] & 0xFu) | (((unsigned)v[1] & 0xFu) << 4));
      }
    }
  }
  return 0;
}

/* Stream id of one weight matrix. matrix: 0 gate, 1 up, 2 down, 3 router. */
uint64_t synth_weight_stream(int64_t layer, int64_t expert, int64_t matrix) {
  return ((uint64_t)layer << 24) | ((uint64_t)expert << 4) | (uint64_t)matrix;
}

/*
 * One weight matrix of `rows` x `cols` (row-major, out x in), values
 * N(0, std = 1/sqrt(fan_in)) in fp32 with fan_in = cols.
 *   wdtype 0: fp32 into out (rows*cols floats)
 *   wdtype 1: bf16 into out (rows*cols uint16)
 *   wdtype 2: int4 g128 into out (rows*cols/2 bytes) + scales (rows*cols/128 bf16)
 * tmp must hold rows*cols floats (unused for wdtype 0).
 */
int synth_weight(uint64_t seed, int64_t layer, int64_t expert, int64_t matrix, int64_t rows, int64_t cols,
                 int wdtype, void* out, uint16_t* scales, float* tmp) {
  float std = (float)(1.0 / sqrt((double)cols));
  uint64_t stream = synth_weight_stream(layer, expert, matrix);
  int64_t n = rows * cols;
  if (wdtype == 0) {
    synth_normal(seed, stream, 0, n, std, (float*)out);
    return 0;
  }
  synth_normal(seed, stream, 0, n, std, tmp);
  if (wdtype == 1) {
    synth_f32_to_bf16(tmp, (uint16_t*)out, n);
    return 0;
  }
  if (wdtype == 2) return synth_quant_int4_g128(tmp, rows, cols, (uint8_t*)out, scales);
  return -1;
}
