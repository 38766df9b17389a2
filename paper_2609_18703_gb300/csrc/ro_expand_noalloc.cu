// ro_expand_noalloc.cu — expansion lineage (offsets, parent and ordinal of
// every child) for callers that cannot allocate device memory.
//
// Some callers cannot call cudaMalloc: code running inside a memory budget
// that a framework's caching allocator owns, code paths that must not
// synchronise the device the way cudaMalloc/cudaFree can, or embedders that
// forbid allocation after start-up.  This entry point needs no context and
// allocates nothing: its scratch (the scan's per-tile look-back status, the
// per-fill-tile parent table and a few counters) lives in one file-scope
// __device__ array of fixed size, which every GPU that loads the library
// holds until the process exits.
//
// Its kernels are variants of expand_scan / expand_fill that write only the
// caller's outputs (no lineage state is kept, so nothing later can commit or
// assemble against this expansion).
#include <cstddef>
#include <mutex>

#include "../../include/rayorch_gpu.h"
#include "ro_internal.h"

namespace ro {
namespace {

constexpr uint64_t NA_MAX_PARENTS = 1ull << 24;    // 16,777,216
constexpr uint64_t NA_MAX_CHILDREN = 1ull << 27;   // 134,217,728
constexpr uint64_t NA_SCAN_TILE = (uint64_t)EXP_THREADS * EXP_ITEMS;
constexpr uint64_t NA_TILES = NA_MAX_PARENTS / NA_SCAN_TILE;        // 4096
constexpr uint64_t NA_TFP = NA_MAX_CHILDREN / FILL_TILE + 1;         // 32769

// Layout of the static scratch.  The header's counters are cleared by every
// call; the epoch is not (it keeps stale tile flags from looking current).
struct NaHeader {
  uint32_t tile_ctr, exit_ctr, err, pad;
  unsigned long long n_children, n_empty, epoch;
};
constexpr size_t NA_OFF_FLAGS = 256;
constexpr size_t NA_OFF_AGG = NA_OFF_FLAGS + NA_TILES * sizeof(unsigned long long);
constexpr size_t NA_OFF_INC = NA_OFF_AGG + NA_TILES * sizeof(Pair64);
constexpr size_t NA_OFF_TFP = NA_OFF_INC + NA_TILES * sizeof(Pair64);
constexpr size_t NA_BYTES = NA_OFF_TFP + NA_TFP * sizeof(uint32_t);   // ~292 KB

static __device__ __align__(256) unsigned char g_expand_scratch[NA_BYTES];

__global__ void __launch_bounds__(EXP_THREADS)
expand_scan_noalloc_kernel(const uint32_t* counts, uint64_t P, uint64_t* offsets,
                           uint32_t* empty_out, unsigned char* scratch) {
  __shared__ Pair64 s_scan[33];
  __shared__ uint32_t s_tile;
  __shared__ Pair64 s_prefix;
  NaHeader* h = reinterpret_cast<NaHeader*>(scratch);
  TileStatus<Pair64> ts{reinterpret_cast<unsigned long long*>(scratch + NA_OFF_FLAGS),
                        reinterpret_cast<Pair64*>(scratch + NA_OFF_AGG),
                        reinterpret_cast<Pair64*>(scratch + NA_OFF_INC)};
  uint32_t* tfp = reinterpret_cast<uint32_t*>(scratch + NA_OFF_TFP);
  const unsigned long long epoch = h->epoch;
  const uint64_t n_tiles = ceil_div(P, NA_SCAN_TILE);
  for (;;) {
    if (threadIdx.x == 0) s_tile = atomicAdd(&h->tile_ctr, 1u);
    __syncthreads();
    const uint32_t tile = s_tile;
    __syncthreads();
    if (tile >= n_tiles) break;
    const uint64_t p0 = tile * NA_SCAN_TILE + (uint64_t)threadIdx.x * EXP_ITEMS;
    uint32_t cnt[EXP_ITEMS];
    Pair64 mine{0, 0};
#pragma unroll
    for (int k = 0; k < EXP_ITEMS; ++k) {
      const uint64_t p = p0 + k;
      cnt[k] = (p < P) ? __ldg(counts + p) : 0u;
      mine.a += cnt[k];
      mine.b += (p < P && cnt[k] == 0u) ? 1ull : 0ull;
    }
    Pair64 total;
    Pair64 excl = block_excl_scan_pair(mine, s_scan, &total);
    if (threadIdx.x < 32) {  // one warp looks back
      const auto pfx = lookback_exclusive(ts, tile, total, epoch, &h->err);
      if (threadIdx.x == 0) s_prefix = pfx;
    }
    __syncthreads();
    Pair64 run = s_prefix + excl;
#pragma unroll
    for (int k = 0; k < EXP_ITEMS; ++k) {
      const uint64_t p = p0 + k;
      if (p >= P) break;
      const uint64_t o = run.a, m = cnt[k];
      offsets[p] = o;
      if (m == 0) {
        if (empty_out) empty_out[run.b] = (uint32_t)p;
        run.b += 1;
      } else {
        for (uint64_t b = ceil_div(o, FILL_TILE); b * FILL_TILE < o + m && b < NA_TFP; ++b)
          tfp[b] = (uint32_t)p;
      }
      run.a += m;
    }
    if (tile == n_tiles - 1 && threadIdx.x == EXP_THREADS - 1) {
      offsets[P] = run.a;
      h->n_children = run.a;
      h->n_empty = run.b;
    }
  }
  if (threadIdx.x == 0) {
    if (n_tiles == 0 && blockIdx.x == 0) {
      offsets[0] = 0;
      h->n_children = 0;
      h->n_empty = 0;
    }
    if (ticket(&h->exit_ctr) == gridDim.x - 1) {
      h->tile_ctr = 0u;
      h->exit_ctr = 0u;
      h->epoch = epoch + 1ull;
    }
  }
}

__global__ void __launch_bounds__(FILL_THREADS)
expand_fill_noalloc_kernel(const uint64_t* offsets, uint64_t P, uint64_t N, uint32_t* child_parent,
                           uint32_t* child_ordinal, const unsigned char* scratch) {
  __shared__ uint64_t s_off[FILL_SMEM_CAP];
  const uint32_t* tfp = reinterpret_cast<const uint32_t*>(scratch + NA_OFF_TFP);
  const uint64_t n_tiles = ceil_div(N, FILL_TILE);
  for (uint64_t t = blockIdx.x; t < n_tiles; t += gridDim.x) {
    const uint64_t c0 = t * FILL_TILE, c1 = min(c0 + FILL_TILE, N);
    const uint64_t p_lo = tfp[t];
    const uint64_t p_hi = (t + 1 < n_tiles) ? tfp[t + 1] : P - 1;
    const uint64_t R = p_hi - p_lo + 2;
    const bool staged = R <= FILL_SMEM_CAP;
    if (staged)
      for (uint64_t k = threadIdx.x; k < R; k += blockDim.x) s_off[k] = offsets[p_lo + k];
    __syncthreads();
    for (uint64_t c = c0 + threadIdx.x; c < c1; c += blockDim.x) {
      uint64_t lo, hi;
      if (staged) {
        uint32_t a = 0, b = (uint32_t)R - 1u;
        while (b - a > 1) {
          const uint32_t mid = a + ((b - a) >> 1);
          if (s_off[mid] <= c) a = mid; else b = mid;
        }
        lo = p_lo + a;
        hi = s_off[a];
      } else {
        uint64_t a = p_lo, b = p_hi + 1;
        while (b - a > 1) {
          const uint64_t mid = a + ((b - a) >> 1);
          if (offsets[mid] <= c) a = mid; else b = mid;
        }
        lo = a;
        hi = offsets[a];
      }
      child_parent[c] = (uint32_t)lo;
      child_ordinal[c] = (uint32_t)(c - hi);
    }
    __syncthreads();
  }
}

// Device address of the static scratch, looked up once per device.
constexpr int NA_MAX_DEVICES = 64;
std::mutex g_na_mu;
unsigned char* g_na_ptr[NA_MAX_DEVICES] = {};
int g_na_sms[NA_MAX_DEVICES] = {};

ro_status na_setup(int dev, unsigned char** ptr, int* sms) {
  if (dev < 0 || dev >= NA_MAX_DEVICES) return RO_E_CUDA;
  std::lock_guard<std::mutex> lock(g_na_mu);
  if (!g_na_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_expand_scratch) != cudaSuccess || !p) {
      cudaGetLastError();
      return RO_E_CUDA;
    }
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1) {
      cudaGetLastError();
      return RO_E_CUDA;
    }
    g_na_ptr[dev] = static_cast<unsigned char*>(p);
    g_na_sms[dev] = n;
  }
  *ptr = g_na_ptr[dev];
  *sms = g_na_sms[dev];
  return RO_OK;
}

}  // namespace
}  // namespace ro

extern "C" ro_status ro_expand_noalloc(const uint32_t* d_counts, uint64_t n_parents,
                                       uint64_t* d_offsets, uint32_t* d_child_parent,
                                       uint32_t* d_child_ordinal, uint64_t child_cap,
                                       uint32_t* d_empty_parents, void* stream,
                                       uint64_t* h_n_children, uint64_t* h_n_empty) {
  using namespace ro;
  if (!h_n_children || !d_offsets || (n_parents && !d_counts)) return RO_E_INVAL;
  if (n_parents > NA_MAX_PARENTS) return RO_E_CAPACITY;   // beyond the static scratch
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return RO_E_CUDA;
  }
  unsigned char* scratch = nullptr;
  int sms = 0;
  ro_status st = na_setup(dev, &scratch, &sms);
  if (st != RO_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // counters must start at zero (the epoch is kept)
  if (cudaMemsetAsync(scratch, 0, offsetof(NaHeader, n_children), s) != cudaSuccess) {
    cudaGetLastError();
    return RO_E_CUDA;
  }
  expand_scan_noalloc_kernel<<<sms * 2, EXP_THREADS, 0, s>>>(d_counts, n_parents, d_offsets,
                                                            d_empty_parents, scratch);
  if (cudaGetLastError() != cudaSuccess) return RO_E_CUDA;   // not launched: the header is stale
  NaHeader hh{};
  cudaError_t e = cudaMemcpyAsync(&hh, scratch, sizeof(NaHeader), cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return RO_E_CUDA;
  }
  *h_n_children = hh.n_children;
  if (h_n_empty) *h_n_empty = hh.n_empty;
  if (hh.err & ERR_TIMEOUT) return RO_E_TIMEOUT;
  const uint64_t N = hh.n_children;
  if (N >= (1ull << 32)) return RO_E_OVERFLOW;
  if (N > NA_MAX_CHILDREN) return RO_E_CAPACITY;   // beyond the static scratch
  if (N > child_cap) return RO_E_CAPACITY;
  if (N == 0) return RO_OK;
  if (!d_child_parent || !d_child_ordinal) return RO_E_INVAL;
  const uint64_t n_tiles = ceil_div(N, FILL_TILE);
  const int grid = (int)(n_tiles < (uint64_t)sms * 8 ? n_tiles : (uint64_t)sms * 8);
  expand_fill_noalloc_kernel<<<grid, FILL_THREADS, 0, s>>>(d_offsets, n_parents, N, d_child_parent,
                                                          d_child_ordinal, scratch);
  if (cudaGetLastError() != cudaSuccess) return RO_E_CUDA;
  // The fill reads the shared scratch (its per-tile parent table): return
  // only once it is done, so that a caller who takes the return as
  // completion may start the next call from any stream or thread.
  if (cudaStreamSynchronize(s) != cudaSuccess) {
    cudaGetLastError();
    return RO_E_CUDA;
  }
  return RO_OK;
}
