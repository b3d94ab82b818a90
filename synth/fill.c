/*
 * Bulk fill for the seeded synthetic inputs (weights, prefix K/V).
 *
 * Generator: SplitMix64 (S. Vigna, "Further scramblings of Marsaglia's
 * xorshift generators", 2015; also the seeding generator of java.util.
 * SplittableRandom), used as a counter-based generator: element i of a stream
 * with key s0 is mix(s0 + (i + 1) * 0x9E3779B97F4A7C15).  Because an element is
 * a pure function of (key, i), any sub-range of a tensor can be generated on
 * its own and is bit-identical to the same range of a full fill.
 *
 * Approximate normal deviate: Irwin-Hall sum of the four 16-bit fields of one
 * 64-bit output, centred (mean 4 * 65535 / 2) and multiplied by `scale` in
 * fp32 (scale = std / sqrt((2^32 - 1) / 3), the exact standard deviation of
 * the sum), then rounded to bf16 with round-to-nearest-even.
 *
 * This file holds input generation only; none of the decoder's arithmetic.
 * Plain C, no intrinsics, so it gives the same bytes on x86-64 and aarch64.
 */
#include <pthread.h>
#include <stddef.h>
#include <stdint.h>
#include <string.h>

#define SM64_GAMMA 0x9E3779B97F4A7C15ULL

static inline uint64_t sm64_mix(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

static inline uint16_t f32_to_bf16_rne(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  u += 0x7FFFu + ((u >> 16) & 1u); /* inputs are finite: no NaN handling needed */
  return (uint16_t)(u >> 16);
}

static inline uint16_t normal_bf16(uint64_t key, uint64_t i, float scale) {
  uint64_t z = sm64_mix(key + (i + 1) * SM64_GAMMA);
  int32_t s = (int32_t)(z & 0xFFFF) + (int32_t)((z >> 16) & 0xFFFF) +
              (int32_t)((z >> 32) & 0xFFFF) + (int32_t)(z >> 48);
  float c = (float)(s - 131070); /* exact: |s - 131070| < 2^24 */
  return f32_to_bf16_rne(c * scale);
}

typedef struct {
  uint64_t key, start;
  size_t count;
  float scale;
  uint16_t* out;
} fill_job;

static void* fill_worker(void* p) {
  fill_job* j = (fill_job*)p;
  for (size_t k = 0; k < j->count; ++k) j->out[k] = normal_bf16(j->key, j->start + k, j->scale);
  return NULL;
}

/* out[k] = bf16 normal deviate of element (start + k) of stream `key`, k < count. */
void synth_fill_normal_bf16(uint64_t key, uint64_t start, size_t count, float scale, uint16_t* out,
                            int threads) {
  if (threads < 1) threads = 1;
  if (threads > 64) threads = 64;
  if (count < (size_t)1 << 20) threads = 1;
  pthread_t tid[64];
  fill_job jobs[64];
  size_t per = (count + (size_t)threads - 1) / (size_t)threads;
  int launched = 0;
  for (int t = 0; t < threads; ++t) {
    size_t b = (size_t)t * per;
    if (b >= count) break;
    size_t e = b + per < count ? b + per : count;
    jobs[t].key = key;
    jobs[t].start = start + b;
    jobs[t].count = e - b;
    jobs[t].scale = scale;
    jobs[t].out = out + b;
    if (threads == 1 || pthread_create(&tid[t], NULL, fill_worker, &jobs[t]) != 0) {
      fill_worker(&jobs[t]);
      tid[t] = 0;
    }
    launched = t + 1;
  }
  for (int t = 0; t < launched; ++t)
    if (tid[t]) pthread_join(tid[t], NULL);
}
