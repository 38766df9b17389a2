// k_expand.cu — ro_expand kernels (Section 4.2; Table 2 child key; Eq. 1).
//
// expand_scan: single-pass exclusive scan of the child counts with
//   decoupled look-back over tiles of 4096 parents.  Alongside the offsets it
//   initialises each parent's terminal counter (remaining = count), lists
//   the empty parents (a second prefix sum carried in the same scan), and
//   records for every fill tile (4096 children) the parent of its first child,
//   so that the fill needs no search in global memory.
// expand_fill: one CTA per 4096-child tile stages the offsets of the parents
//   that tile touches in shared memory and gives every child its parent (a
//   binary search in shared memory) and ordinal; it also initialises the
//   child's Grain phase (WAITING, unclaimed) and result record.  Work per CTA
//   is bounded by the tile, so one 100k-child parent spreads over 25 tiles
//   instead of serialising a warp.
#include <algorithm>

#include "ro_internal.h"

namespace ro {

__global__ void __launch_bounds__(EXP_THREADS) expand_scan_kernel(ExpandScanArgs a) {
  wait_predecessor();
  __shared__ Pair64 s_scan[33];
  __shared__ uint32_t s_tile;
  __shared__ Pair64 s_prefix;
  const uint64_t TILE = (uint64_t)EXP_THREADS * EXP_ITEMS;
  const uint64_t n_tiles = ceil_div(a.P, TILE);
  DevScalars* ds = a.ds;
  if (n_tiles == 0) {
    if (blockIdx.x == 0 && threadIdx.x == 0) {
      a.offsets_user[0] = 0;
      a.offsets[0] = 0;
      ds->n_children = 0;
      ds->n_empty = 0;
    }
    return;
  }
  const uint32_t n_part = participants(n_tiles);
  if (blockIdx.x >= n_part) return;

  for (;;) {
    if (threadIdx.x == 0) s_tile = claim_tile(&ds->tile_ctr[TS_EXPAND]);
    __syncthreads();
    const uint32_t tile = s_tile;
    __syncthreads();
    if (tile >= n_tiles) break;

    const uint64_t p0 = tile * TILE + (uint64_t)threadIdx.x * EXP_ITEMS;
    uint32_t cnt[EXP_ITEMS];
    Pair64 mine{0, 0};
#pragma unroll
    for (int k = 0; k < EXP_ITEMS; ++k) {
      const uint64_t p = p0 + k;
      cnt[k] = (p < a.P) ? __ldg(a.counts + p) : 0u;
      mine.a += cnt[k];
      mine.b += (p < a.P && cnt[k] == 0u) ? 1ull : 0ull;
    }
    unsigned long long heavy = 0;   // children of heavy parents
#pragma unroll
    for (int k = 0; k < EXP_ITEMS; ++k) heavy += cnt[k] >= HEAVY_CHILDREN ? cnt[k] : 0u;
    for (int d = 16; d > 0; d >>= 1) heavy += __shfl_xor_sync(0xffffffffu, heavy, d);
    if ((threadIdx.x & 31) == 0 && heavy) atomicAdd(&ds->n_heavy, heavy);
    Pair64 total;
    Pair64 excl = block_excl_scan_pair(mine, s_scan, &total);
    if (threadIdx.x < 32) {  // one warp looks back
      const auto pfx = lookback_exclusive(a.ts, tile, total, ds->epoch[TS_EXPAND], &ds->err);
      if (threadIdx.x == 0) s_prefix = pfx;
    }
    __syncthreads();
    Pair64 run = s_prefix + excl;
#pragma unroll
    for (int k = 0; k < EXP_ITEMS; ++k) {
      const uint64_t p = p0 + k;
      if (p >= a.P) break;
      const uint64_t o = run.a, m = cnt[k];
      a.offsets_user[p] = o;
      a.offsets[p] = o;
      a.pw[p] = m;   // remaining = count, bad = 0
      if (m == 0) {
        if (a.empty_out) a.empty_out[run.b] = (uint32_t)p;
        run.b += 1;
      } else {
        // fill tiles whose first child is a child of p
        for (uint64_t b = ceil_div(o, FILL_TILE); b * FILL_TILE < o + m && b < a.tfp_cap; ++b)
          a.tfp[b] = (uint32_t)p;
      }
      run.a += m;
    }
    if (tile == n_tiles - 1 && threadIdx.x == EXP_THREADS - 1) {
      a.offsets_user[a.P] = run.a;
      a.offsets[a.P] = run.a;
      ds->n_children = run.a;
      ds->n_empty = run.b;
    }
  }
  if (threadIdx.x == 0) retire_cta(ds, TS_EXPAND, n_part);
}

// Largest index k in [lo, hi) with v[k] <= x (v non-decreasing, v[lo] <= x).
template <class V>
__device__ __forceinline__ uint32_t last_le(const V* v, uint32_t lo, uint32_t hi, uint64_t x) {
  while (hi - lo > 1) {
    const uint32_t mid = lo + ((hi - lo) >> 1);
    if ((uint64_t)v[mid] <= x)
      lo = mid;
    else
      hi = mid;
  }
  return lo;
}

__global__ void __launch_bounds__(FILL_THREADS) expand_fill_kernel(ExpandFillArgs a) {
  wait_predecessor();
  __shared__ uint64_t s_off[FILL_SMEM_CAP];
  const uint64_t n_tiles = ceil_div(a.N, FILL_TILE);
  for (uint64_t t = blockIdx.x; t < n_tiles; t += gridDim.x) {
    const uint64_t c0 = t * FILL_TILE, c1 = min(c0 + FILL_TILE, a.N);
    const uint64_t p_lo = a.tfp[t];
    const uint64_t p_hi = (t + 1 < n_tiles) ? a.tfp[t + 1] : a.P - 1;
    const uint64_t R = p_hi - p_lo + 2;   // offsets[p_lo .. p_hi+1]
    const bool staged = R <= FILL_SMEM_CAP;
    if (staged) {
      for (uint64_t k = threadIdx.x; k < R; k += blockDim.x) s_off[k] = a.offsets[p_lo + k];
    }
    __syncthreads();
    for (uint64_t c = c0 + threadIdx.x; c < c1; c += blockDim.x) {
      uint64_t p, base;
      if (staged) {
        const uint32_t k = last_le(s_off, 0u, (uint32_t)R - 1u, c);
        p = p_lo + k;
        base = s_off[k];
      } else {
        // many empty parents inside one tile: search the global offsets
        uint64_t lo = p_lo, hi = p_hi + 1;
        while (hi - lo > 1) {
          const uint64_t mid = lo + ((hi - lo) >> 1);
          if (a.offsets[mid] <= c)
            lo = mid;
          else
            hi = mid;
        }
        p = lo;
        base = a.offsets[lo];
      }
      const uint32_t call = a.parent_call ? (uint32_t)a.parent_call[p] : 0u;
      a.child_parent[c] = (uint32_t)p;
      a.child_ordinal[c] = (uint32_t)(c - base);
      a.par[c] = (uint32_t)p;
      Slot sl;
      sl.phase = WAIT_UNCLAIMED;
      sl.len = 0u;
      sl.w = (uint64_t)call << W_CALL_SHIFT;
      a.slot[c] = sl;
    }
    __syncthreads();
  }
}

void launch_expand_scan(const LaunchCfg& L, const ExpandScanArgs& a) {
  launch_k(L, K_EXPAND_SCAN, expand_scan_kernel, L.grid_expand_scan, EXP_THREADS, 0, a);
}

void launch_expand_fill(const LaunchCfg& L, const ExpandFillArgs& a) {
  const uint64_t n_tiles = ceil_div(a.N, FILL_TILE);
  if (n_tiles == 0) return;
  const int grid = (int)std::min<uint64_t>(n_tiles, (uint64_t)L.grid_fill);
  launch_k(L, K_FILL, expand_fill_kernel, grid, FILL_THREADS, 0, a);
}

const void* kernel_ptr_expand(int which) {
  return which == K_EXPAND_SCAN ? (const void*)expand_scan_kernel : (const void*)expand_fill_kernel;
}

}  // namespace ro
