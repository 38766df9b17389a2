// payload_fill.cu — device-side fill of synthetic result payloads.
//
// Writes, for every child c with len[c] > 0, the record defined in
// workload/payload.py: byte j is byte (j & 7) of mix64(seed ^ c*GOLDEN +
// (j >> 3)*WORDSTEP), mix64 being the SplitMix64 finaliser (Steele, Lea and
// Flood, OOPSLA 2014).  Input generation only; no lineage arithmetic.
#include <cstdint>
#include <cuda_runtime.h>

namespace {
constexpr uint64_t GOLDEN = 0x9E3779B97F4A7C15ull;
constexpr uint64_t WORDSTEP = 0xD1B54A32D192ED03ull;

__device__ __forceinline__ uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// one warp per record; lane l writes bytes l, l+32, ... (each warp store is
// 32 consecutive bytes)
__global__ void fill_kernel(uint8_t* arena, uint64_t arena_bytes, const uint64_t* off,
                            const uint32_t* len, uint64_t n, uint64_t seed) {
  const uint64_t lane = threadIdx.x & 31;
  const uint64_t warp = ((uint64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const uint64_t n_warps = ((uint64_t)gridDim.x * blockDim.x) >> 5;
  for (uint64_t c = warp; c < n; c += n_warps) {
    const uint64_t L = len[c], o = off[c];
    if (L == 0 || o > arena_bytes || L > arena_bytes - o) continue;
    const uint64_t base = seed ^ (c * GOLDEN);
    for (uint64_t b = lane; b < L; b += 32) {
      const uint64_t z = mix64(base + (b >> 3) * WORDSTEP);
      arena[o + b] = (uint8_t)(z >> (8 * (b & 7)));
    }
  }
}
}  // namespace

extern "C" int wl_fill_payload(uint8_t* arena, uint64_t arena_bytes, const uint64_t* off,
                               const uint32_t* len, uint64_t n_children, uint64_t seed,
                               void* stream) {
  if (n_children == 0) return 0;
  int sms = 0, dev = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const uint64_t want = (n_children + 7) / 8;
  const int grid = (int)(want < (uint64_t)sms * 16 ? (want ? want : 1) : (uint64_t)sms * 16);
  fill_kernel<<<grid, 256, 0, (cudaStream_t)stream>>>(arena, arena_bytes, off, len, n_children, seed);
  return (int)cudaGetLastError();
}
