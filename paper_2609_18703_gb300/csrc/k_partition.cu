// k_partition.cu — a large commit's reports grouped by child range before
// the fence (Section 4.4, Eq. 3; Section 4.2, Reduce).
//
// The commit's scatter touches each report's slot, parent and parent
// counter.  Tens of millions of reports in random order make each of those a
// DRAM round trip.  Grouped by child range first — PT_BUCKETS ranges of
// about N / PT_BUCKETS children, whose edges fall on parent boundaries — the
// scatter, which walks the grouped reports in order, works on one range's
// slots and counters at a time, and those stay in L2.  The grouping is
// stable and never splits a parent's children, so the reports of one parent
// (and so of one child) keep their relative array order: the rules of a
// commit that depend on order (the first of several reports of a Grain wins;
// a GroupFailure bars its siblings' later reports) compare a report only
// with reports of the same parent, and decide on the grouped array as on the
// caller's.
//   part_hist       per tile of PT_TILE reports, the count of each range
//                   (and each range's total);
//   part_scan       per range, where each tile's reports of that range start
//                   (one CTA per range);
//   part_scatter    each tile's reports moved to their ranges, in array order
//                   within the tile, tile after tile;
//   part_unpermute  the verdict codes back in the caller's order (only when
//                   the caller asked for them).
#include <algorithm>
#include <type_traits>

#include "ro_internal.h"

namespace ro {

namespace {

static_assert(PT_THREADS == PT_BUCKETS, "one range per thread in the per-range steps");
constexpr int PT_WARPS = PT_THREADS / 32;
constexpr int PT_SCAN_ITEMS = 8;

__device__ __forceinline__ uint64_t part_count(const PartArgs& a) {
  if (!a.d_n) return a.n_host;
  const uint64_t n = *a.d_n;
  return n < a.n_host ? n : a.n_host;
}

// Range edges.  Edge k (0 < k < PT_BUCKETS) is the first child of the parent
// holding child (k * n_fill_tiles / PT_BUCKETS) * FILL_TILE, from the fill-tile
// table and the offsets: non-decreasing in k, and the first child of a
// parent that has children, so never strictly inside a parent's children.
// Edge 0 is 0.
__device__ __forceinline__ uint32_t edge_of(const PartArgs& a, uint32_t k) {
  if (k == 0 || a.n_fill_tiles == 0) return 0u;
  const uint64_t t = (uint64_t)k * a.n_fill_tiles / PT_BUCKETS;   // < n_fill_tiles
  return (uint32_t)a.offsets[a.tfp[t]];
}

// The range of child c: the last k with edge k <= c.  A child id past the
// expansion falls in the last range (its report is rejected as invalid).
__device__ __forceinline__ uint32_t range_of(const uint32_t* s_edge, uint32_t c) {
  uint32_t k = 0;
#pragma unroll
  for (uint32_t step = PT_BUCKETS / 2; step > 0; step >>= 1)
    if (s_edge[k + step] <= c) k += step;
  return k;
}

}  // namespace

__global__ void __launch_bounds__(PT_THREADS) part_hist_kernel(PartArgs a) {
  __shared__ uint32_t s_edge[PT_BUCKETS];
  __shared__ uint32_t s_hist[PT_BUCKETS];
  wait_predecessor();
  allow_successor();
  s_edge[threadIdx.x] = edge_of(a, threadIdx.x);
  if (blockIdx.x == 0) a.edges[threadIdx.x] = s_edge[threadIdx.x];   // for part_scatter
  const uint64_t n = part_count(a);
  constexpr int R = PT_TILE / PT_THREADS;
  for (uint64_t t = blockIdx.x; t < a.n_tiles; t += gridDim.x) {
    s_hist[threadIdx.x] = 0u;
    __syncthreads();
    const uint64_t r0 = t * PT_TILE + threadIdx.x;
    uint32_t cv[R];
#pragma unroll
    for (int j = 0; j < R; ++j) {   // all of this thread's children in flight at once
      const uint64_t r = r0 + (uint64_t)j * PT_THREADS;
      cv[j] = r < n ? a.child[r] : 0u;
    }
#pragma unroll
    for (int j = 0; j < R; ++j)
      if (r0 + (uint64_t)j * PT_THREADS < n) atomicAdd(&s_hist[range_of(s_edge, cv[j])], 1u);
    __syncthreads();
    const uint32_t h = s_hist[threadIdx.x];
    a.hist[(uint64_t)threadIdx.x * a.n_tiles + t] = h;
    if (h) atomicAdd(&a.btot[threadIdx.x], h);
    __syncthreads();   // s_hist is zeroed for the next tile only after every read
  }
}

// One CTA per range b: the range starts after the ranges before it; inside
// it, tile t's reports start after those of the tiles before t.
__global__ void __launch_bounds__(PT_THREADS) part_scan_kernel(PartArgs a) {
  __shared__ unsigned long long s_scan[33];
  wait_predecessor();
  allow_successor();
  const uint32_t b = blockIdx.x;
  unsigned long long carry;
  block_excl_scan<unsigned long long>(threadIdx.x < b ? (unsigned long long)a.btot[threadIdx.x] : 0ull,
                                      s_scan, &carry);
  const uint32_t* h = a.hist + (uint64_t)b * a.n_tiles;
  uint32_t* o = a.pfx + (uint64_t)b * a.n_tiles;
  for (uint64_t t0 = 0; t0 < a.n_tiles; t0 += (uint64_t)PT_THREADS * PT_SCAN_ITEMS) {
    const uint64_t tb = t0 + (uint64_t)threadIdx.x * PT_SCAN_ITEMS;
    uint32_t x[PT_SCAN_ITEMS];
    unsigned long long s = 0;
#pragma unroll
    for (int k = 0; k < PT_SCAN_ITEMS; ++k) {
      x[k] = (tb + k < a.n_tiles) ? h[tb + k] : 0u;
      s += x[k];
    }
    unsigned long long chunk;
    unsigned long long p = carry + block_excl_scan<unsigned long long>(s, s_scan, &chunk);
#pragma unroll
    for (int k = 0; k < PT_SCAN_ITEMS; ++k) {
      if (tb + k < a.n_tiles) o[tb + k] = (uint32_t)p;
      p += x[k];
    }
    carry += chunk;
  }
}

// Each tile's reports, in rounds of PT_THREADS in array order: a report's
// place in its range is the range's start for this tile plus the reports of
// that range placed by earlier rounds, by earlier warps of this round and by
// earlier lanes of its warp (__match_any_sync).  The tile's reports are
// first ordered by range in shared memory (each one's tile index and
// destination), then every field is staged from the caller's array and
// written out in that order, so consecutive threads write consecutive places
// of a range.
__global__ void __launch_bounds__(PT_THREADS) part_scatter_kernel(PartArgs a) {
  __shared__ uint32_t s_edge[PT_BUCKETS];
  __shared__ uint32_t s_gbase[PT_BUCKETS];            // per range: first place of this tile's reports
  __shared__ uint32_t s_tro[PT_BUCKETS];              // per range: its first position in the tile's order
  __shared__ uint32_t s_next[PT_BUCKETS];             // per range: reports of the tile placed so far
  __shared__ uint32_t s_cnt[PT_WARPS][PT_BUCKETS];    // per warp and range: reports this round, tagged
  __shared__ uint16_t s_start[PT_WARPS][PT_BUCKETS];  // per warp and range: first rank this round
  __shared__ uint16_t s_src[PT_TILE];                 // by position in the tile's order: tile index
  __shared__ uint32_t s_dst[PT_TILE];                 // by position in the tile's order: destination
  __shared__ uint64_t s_stage[PT_TILE];               // one field of the tile, in array order
  __shared__ uint32_t s_scan[33];
  wait_predecessor();
  allow_successor();
  s_edge[threadIdx.x] = a.edges[threadIdx.x];
#pragma unroll
  for (int w = 0; w < PT_WARPS; ++w) s_cnt[w][threadIdx.x] = 0u;   // tag 0: no round yet
  const uint64_t n = part_count(a);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const unsigned lower = (1u << lane) - 1u;
  uint32_t tag = 0;   // rounds of this CTA, from 1 (a count carries its round in bits 6 and up)
  for (uint64_t t = blockIdx.x; t < a.n_tiles; t += gridDim.x) {
    const uint64_t r0 = t * PT_TILE;
    const uint32_t cnt = (uint32_t)(n > r0 ? (n - r0 < PT_TILE ? n - r0 : PT_TILE) : 0);
    {   // range threadIdx.x: where this tile's reports of it go, and their place in the tile's order
      const uint64_t hb = (uint64_t)threadIdx.x * a.n_tiles + t;
      const uint32_t h = a.hist[hb];
      s_gbase[threadIdx.x] = a.pfx[hb];
      s_next[threadIdx.x] = 0u;
      uint32_t tot;
      s_tro[threadIdx.x] = block_excl_scan<uint32_t>(h, s_scan, &tot);   // (synchronises the block)
    }
    uint32_t c = threadIdx.x < cnt ? a.child[r0 + threadIdx.x] : 0u;
    for (uint32_t j = 0; j < PT_TILE; j += PT_THREADS) {
      const uint32_t i = j + threadIdx.x;   // tile index
      const bool act = i < cnt;
      const uint32_t cn = (i + PT_THREADS < cnt) ? a.child[r0 + i + PT_THREADS] : 0u;   // next round
      ++tag;
      const uint32_t k = act ? range_of(s_edge, c) : (uint32_t)PT_BUCKETS;   // PT_BUCKETS: no report
      const unsigned peers = __match_any_sync(0xffffffffu, k);
      const uint32_t rank = (uint32_t)__popc(peers & lower);
      if (act && rank == 0) s_cnt[warp][k] = (tag << 6) | (uint32_t)__popc(peers);
      __syncthreads();
      {   // range threadIdx.x: the warps' first ranks this round
        uint32_t next = s_next[threadIdx.x];
#pragma unroll
        for (int w = 0; w < PT_WARPS; ++w) {
          const uint32_t v = s_cnt[w][threadIdx.x];
          s_start[w][threadIdx.x] = (uint16_t)next;
          if ((v >> 6) == tag) next += v & 63u;
        }
        s_next[threadIdx.x] = next;
      }
      __syncthreads();
      if (act) {
        const uint32_t q = (uint32_t)s_start[warp][k] + rank;   // rank in the range, in this tile
        const uint32_t lp = s_tro[k] + q;
        if (lp < cnt) {
          s_src[lp] = (uint16_t)i;
          s_dst[lp] = s_gbase[k] + q;
        }
      }
      c = cn;
    }
    __syncthreads();
    // the fields, staged in array order and written in the tile's order
    auto move = [&](auto* dst, const auto* src) {
      for (uint32_t i = threadIdx.x; i < cnt; i += PT_THREADS) s_stage[i] = (uint64_t)src[r0 + i];
      __syncthreads();
      for (uint32_t lp = threadIdx.x; lp < cnt; lp += PT_THREADS) {
        const uint32_t d = s_dst[lp];
        if (d < n) dst[d] = (std::remove_reference_t<decltype(*dst)>)s_stage[s_src[lp]];
      }
      __syncthreads();
    };
    move(a.child_p, a.child);
    move(a.state_p, a.state);
    move(a.len_p, a.len);
    move(a.off_p, a.off);
    if (a.gen_p) move(a.gen_p, a.gen);
    if (a.rix_p)
      for (uint32_t lp = threadIdx.x; lp < cnt; lp += PT_THREADS) {
        const uint32_t d = s_dst[lp];
        if (d < n) a.rix_p[d] = (uint32_t)(r0 + s_src[lp]);
      }
    __syncthreads();   // s_src and s_dst are rewritten by the next tile
  }
}

// The verdicts back in the caller's order.
__global__ void __launch_bounds__(PT_THREADS) part_unpermute_kernel(PartArgs a) {
  wait_predecessor();
  allow_successor();
  const uint64_t n = part_count(a);
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  for (uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
    const uint32_t r = a.rix_p[i];
    if (r < n) a.code_out[r] = a.code_p[i];
  }
}

void launch_partition(const LaunchCfg& L, const PartArgs& a) {
  const int grid = (int)std::max<uint64_t>(1, std::min<uint64_t>(a.n_tiles, (uint64_t)L.grid_commit));
  launch_k(L, K_PT_HIST, part_hist_kernel, grid, PT_THREADS, 0, a);
  launch_k(L, K_PT_SCAN, part_scan_kernel, PT_BUCKETS, PT_THREADS, 0, a);
  launch_k(L, K_PT_SCATTER, part_scatter_kernel, grid, PT_THREADS, 0, a);
}

void launch_unpermute(const LaunchCfg& L, const PartArgs& a) {
  const int grid = (int)std::max<uint64_t>(
      1, std::min<uint64_t>(ceil_div(a.n_host, (uint64_t)PT_THREADS), (uint64_t)L.grid_commit));
  launch_k(L, K_PT_UNPERM, part_unpermute_kernel, grid, PT_THREADS, 0, a);
}

}  // namespace ro
