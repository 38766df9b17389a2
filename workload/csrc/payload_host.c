/* payload_host.c — host-side fill of synthetic result payloads (same
 * definition as payload_fill.cu and workload/payload.py: byte j of child c's
 * record is byte (j & 7) of SplitMix64-mix(seed ^ c*GOLDEN + (j >> 3)*WORDSTEP)).
 * Input generation only. */
#include <stdint.h>

static uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

int wl_fill_host(uint8_t* arena, uint64_t arena_bytes, const uint64_t* child, const uint64_t* off,
                 const uint64_t* len, uint64_t n, uint64_t seed) {
  for (uint64_t i = 0; i < n; ++i) {
    const uint64_t L = len[i], o = off[i];
    if (!L) continue;
    if (o > arena_bytes || L > arena_bytes - o) return 1;
    const uint64_t base = seed ^ (child[i] * 0x9E3779B97F4A7C15ull);
    for (uint64_t w = 0; w * 8 < L; ++w) {
      const uint64_t z = mix64(base + w * 0xD1B54A32D192ED03ull);
      for (uint64_t b = 0; b < 8 && w * 8 + b < L; ++b) arena[o + w * 8 + b] = (uint8_t)(z >> (8 * b));
    }
  }
  return 0;
}
