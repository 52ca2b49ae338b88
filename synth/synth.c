/*
 * Seeded synthetic inputs shared by the CUDA path and the CPU oracle.
 *
 * This file holds no arithmetic of the method (no normalisation, projection,
 * rotary embedding or attention). It only draws the random inputs that both
 * sides consume byte for byte:
 *   - weight tensors: N(0, sigma^2) samples rounded to bf16 (round to nearest
 *     even), sigma = 0.02 for the workloads in the paper's setting;
 *   - token ids: uniform over [0, vocab);
 *   - scattered eviction choices: a seeded Fisher-Yates shuffle.
 *
 * Generator: SplitMix64 (Steele, Lea and Flood, "Fast splittable pseudorandom
 * number generators", OOPSLA 2014; the 64-bit finaliser constants are the
 * published ones).  Every output is a pure function of (seed, tensor id,
 * element index), so any slice of a tensor can be generated independently and
 * the result does not depend on the thread count.
 *
 * Normals: Box-Muller transform (Box and Muller, 1958) on two 53-bit uniforms;
 * element 2j takes the cosine branch and element 2j+1 the sine branch.
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

static inline uint64_t sm64(uint64_t x) {
  uint64_t z = x + 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

/* Stream key of one tensor: independent streams per (seed, tensor id). */
uint64_t synth_key(uint64_t seed, uint64_t tensor_id) {
  return sm64(sm64(seed) ^ (tensor_id * 0xD1B54A32D192ED03ull));
}

uint64_t synth_u64(uint64_t key, uint64_t counter) { return sm64(key + counter); }

static inline uint16_t f32_to_bf16_rne(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  uint32_t lsb = (u >> 16) & 1u;
  u += 0x7FFFu + lsb;
  return (uint16_t)(u >> 16);
}

/* One Box-Muller pair at pair index j of stream `key`. */
static inline void normal_pair(uint64_t key, uint64_t j, double* z0, double* z1) {
  uint64_t r1 = sm64(key + 2 * j), r2 = sm64(key + 2 * j + 1);
  double u1 = (double)((r1 >> 11) + 1) * 0x1.0p-53; /* (0, 1] */
  double u2 = (double)(r2 >> 11) * 0x1.0p-53;       /* [0, 1) */
  double rad = sqrt(-2.0 * log(u1));
  double a = 6.283185307179586476925 * u2;
  *z0 = rad * cos(a);
  *z1 = rad * sin(a);
}

/* Elements [begin, begin+n) of tensor (seed, tensor_id): sigma * N(0,1) as bf16. */
void synth_normal_bf16(uint64_t seed, uint64_t tensor_id, double sigma, int64_t begin, int64_t n,
                       uint16_t* out) {
  uint64_t key = synth_key(seed, tensor_id);
#pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < n; ++i) {
    uint64_t e = (uint64_t)(begin + i);
    double z0, z1;
    normal_pair(key, e >> 1, &z0, &z1);
    double z = (e & 1) ? z1 : z0;
    out[i] = f32_to_bf16_rne((float)(sigma * z));
  }
}

/* Same samples as float64 before any rounding (for tests of the generator). */
void synth_normal_f64(uint64_t seed, uint64_t tensor_id, int64_t begin, int64_t n, double* out) {
  uint64_t key = synth_key(seed, tensor_id);
  for (int64_t i = 0; i < n; ++i) {
    uint64_t e = (uint64_t)(begin + i);
    double z0, z1;
    normal_pair(key, e >> 1, &z0, &z1);
    out[i] = (e & 1) ? z1 : z0;
  }
}

/* Token ids uniform over [0, vocab): element i = u64(key, i) mod vocab. */
void synth_tokens(uint64_t seed, uint64_t tensor_id, int64_t n, int32_t vocab, int32_t* out) {
  uint64_t key = synth_key(seed, tensor_id);
  for (int64_t i = 0; i < n; ++i) out[i] = (int32_t)(sm64(key + (uint64_t)i) % (uint64_t)vocab);
}

/* Seeded Fisher-Yates: a uniform random permutation of [0, n) (Durstenfeld's
 * in-place form); the first k entries are a uniform k-subset. */
void synth_permutation(uint64_t seed, uint64_t tensor_id, int64_t n, int64_t* out) {
  uint64_t key = synth_key(seed, tensor_id);
  for (int64_t i = 0; i < n; ++i) out[i] = i;
  for (int64_t i = n - 1; i > 0; --i) {
    uint64_t r = sm64(key + (uint64_t)(n - 1 - i));
    int64_t j = (int64_t)(r % (uint64_t)(i + 1));
    int64_t t = out[i];
    out[i] = out[j];
    out[j] = t;
  }
}

/* 64-bit FNV-1a over bytes: a content fingerprint for comparing tensors. */
uint64_t synth_fnv1a(const void* data, int64_t nbytes) {
  const unsigned char* p = (const unsigned char*)data;
  uint64_t h = 0xcbf29ce484222325ull;
  for (int64_t i = 0; i < nbytes; ++i) {
    h ^= p[i];
    h *= 0x100000001b3ull;
  }
  return h;
}
