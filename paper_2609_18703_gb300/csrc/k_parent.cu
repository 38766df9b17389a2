// k_parent.cu — parent-bound reservation (Section 4.3): each reservation
// takes up to B queued siblings of the parent of the queue's first entry and
// leaves the other entries in order.
//
// Repeated reservations have a closed form, which these kernels compute in
// parallel: rank every queued entry among its parent's queued entries (queue
// order) and cut each parent's entries into chunks of B; the reservations
// take exactly these chunks, in increasing queue position of each chunk's
// first entry (without flush, up to the first chunk shorter than B).  The
// ranks come from a stable sort of the window by parent id.
//
//   pb_keys     window copy: child, parent (sort key), position (sort value);
//               clears the per-position chunk sizes and marks
//   pb_hist     per tile digit counts of one 8-bit digit of the key
//   pb_rowscan  per digit, exclusive scan over tiles; digit totals
//   pb_sort     stable scatter of one digit pass (warp match + per-warp counts)
//   pb_bounds   per parent, sorted range of its entries
//   pb_heads    sorted order: each chunk's first entry records the chunk size
//               at its queue position; the first short chunk (no flush)
//   pb_mark     sorted order, no flush only: marks entries of chunks at or
//               after the first short chunk, which stay queued
//   pb_scan     queue order, single-pass scan (decoupled look-back): output
//               offset of each taken chunk, batch boundaries, entries left
//   pb_emit     sorted order: writes each taken chunk's entries contiguously
//               (IN-FLIGHT) and the queue's remainder, or on a refusal
//               (capacity) undoes the admission
// Only chunk heads (about one entry in B) and marked entries are written by
// queue position; everything else moves in sorted order.
// The admission itself (ready_count / ready_scatter with parent_bound set)
// runs first and queues every admitted Grain.
#include <algorithm>

#include "ro_internal.h"

namespace ro {

__global__ void __launch_bounds__(PB_THREADS) pb_keys_kernel(ParentArgs a) {
  wait_predecessor();
  constexpr int U = 4;   // entries per thread per step: their loads first
  const DevScalars* ds = a.ds;
  const uint64_t Q = ds->pb_Q, head = ds->pb_head;
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  for (uint64_t j0 = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; j0 < Q; j0 += U * stride) {
    uint32_t c[U], p[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const uint64_t j = j0 + u * stride;
      c[u] = j < Q ? a.queue[head + j] : 0u;
    }
#pragma unroll
    for (int u = 0; u < U; ++u) p[u] = j0 + u * stride < Q ? a.par[c[u]] : 0u;
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const uint64_t j = j0 + u * stride;
      if (j >= Q) break;
      a.child[j] = c[u];
      a.key[0][j] = p[u];
      a.val[0][j] = (uint32_t)j;
      a.hsz[j] = 0u;
      a.left[j] = 0u;
    }
  }
}

__device__ __forceinline__ uint64_t pb_tiles(uint64_t Q) { return ceil_div(Q, (uint64_t)PB_TILE); }

__global__ void __launch_bounds__(PB_THREADS) pb_hist_kernel(ParentArgs a) {
  wait_predecessor();
  __shared__ uint32_t s_h[PB_DIGITS];
  const uint64_t Q = a.ds->pb_Q, T = pb_tiles(Q);
  const uint32_t* key = a.key[a.pass & 1];
  const int shift = 8 * a.pass;
  for (uint64_t t = blockIdx.x; t < T; t += gridDim.x) {
    s_h[threadIdx.x] = 0u;
    __syncthreads();
#pragma unroll
    for (int k = 0; k < PB_ITEMS; ++k) {
      const uint64_t i = t * PB_TILE + (uint64_t)k * PB_THREADS + threadIdx.x;
      if (i < Q) atomicAdd(&s_h[(key[i] >> shift) & 255u], 1u);
    }
    __syncthreads();
    a.hist[(uint64_t)threadIdx.x * T + t] = s_h[threadIdx.x];
    __syncthreads();
  }
}

// One CTA per digit: exclusive scan of that digit's counts over the tiles.
__global__ void __launch_bounds__(PB_THREADS) pb_rowscan_kernel(ParentArgs a) {
  wait_predecessor();
  __shared__ uint32_t s_scan[33];
  const uint64_t T = pb_tiles(a.ds->pb_Q);
  uint32_t* row = a.hist + (uint64_t)blockIdx.x * T;
  uint32_t carry = 0;
  for (uint64_t b = 0; b < T; b += PB_THREADS) {
    const uint64_t t = b + threadIdx.x;
    const uint32_t v = t < T ? row[t] : 0u;
    uint32_t total;
    const uint32_t ex = block_excl_scan(v, s_scan, &total);
    if (t < T) row[t] = carry + ex;
    carry += total;
  }
  if (threadIdx.x == 0) a.dtot[blockIdx.x] = carry;
}

// Stable scatter of one digit pass.  Warp w of a tile owns entries
// [w*256, (w+1)*256) of the tile and walks them 32 at a time in order; lanes
// holding the same digit find each other with a warp match and take
// consecutive places after the warp's running count of that digit.  The
// warps' counts are then scanned per digit, so places follow tile order,
// warp order, round order and lane order: the original order.
__global__ void __launch_bounds__(PB_THREADS) pb_sort_kernel(ParentArgs a) {
  wait_predecessor();
  constexpr int NW = PB_THREADS / 32;
  __shared__ uint32_t s_cnt[NW][PB_DIGITS];
  __shared__ uint32_t s_dbase[PB_DIGITS];
  __shared__ uint32_t s_gbase[PB_DIGITS];
  __shared__ uint32_t s_scan[33];
  const uint64_t Q = a.ds->pb_Q, T = pb_tiles(Q);
  const uint32_t* kin = a.key[a.pass & 1];
  const uint32_t* vin = a.val[a.pass & 1];
  uint32_t* kout = a.key[(a.pass + 1) & 1];
  uint32_t* vout = a.val[(a.pass + 1) & 1];
  const int shift = 8 * a.pass;
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  {
    uint32_t tot;
    const uint32_t ex = block_excl_scan(a.dtot[threadIdx.x], s_scan, &tot);
    s_dbase[threadIdx.x] = ex;
  }
  for (uint64_t t = blockIdx.x; t < T; t += gridDim.x) {
    for (int w2 = 0; w2 < NW; ++w2) s_cnt[w2][threadIdx.x] = 0u;
    __syncthreads();
    uint32_t kk[PB_ITEMS], vv[PB_ITEMS], lo[PB_ITEMS];
    const uint64_t base = t * PB_TILE + (uint64_t)w * (32 * PB_ITEMS);
#pragma unroll
    for (int r = 0; r < PB_ITEMS; ++r) {
      const uint64_t i = base + (uint64_t)r * 32 + lane;
      const bool valid = i < Q;
      kk[r] = valid ? kin[i] : 0u;
      vv[r] = valid ? vin[i] : 0u;
      const uint32_t d = valid ? (kk[r] >> shift) & 255u : (uint32_t)PB_DIGITS;
      const uint32_t peers = __match_any_sync(0xffffffffu, d);
      const uint32_t before = __popc(peers & ((1u << lane) - 1u));
      const uint32_t run = valid ? s_cnt[w][d] : 0u;
      __syncwarp();
      if (valid && before == 0u) s_cnt[w][d] = run + __popc(peers);
      __syncwarp();
      lo[r] = run + before;
    }
    __syncthreads();
    {
      const uint32_t d = threadIdx.x;
      uint32_t run = 0;
      for (int w2 = 0; w2 < NW; ++w2) {
        const uint32_t c = s_cnt[w2][d];
        s_cnt[w2][d] = run;
        run += c;
      }
      s_gbase[d] = s_dbase[d] + a.hist[(uint64_t)d * T + t];
    }
    __syncthreads();
#pragma unroll
    for (int r = 0; r < PB_ITEMS; ++r) {
      const uint64_t i = base + (uint64_t)r * 32 + lane;
      if (i >= Q) continue;
      const uint32_t d = (kk[r] >> shift) & 255u;
      const uint32_t o = s_gbase[d] + s_cnt[w][d] + lo[r];
      kout[o] = kk[r];
      vout[o] = vv[r];
    }
    __syncthreads();
  }
}

__global__ void __launch_bounds__(PB_THREADS) pb_bounds_kernel(ParentArgs a) {
  wait_predecessor();
  const uint64_t Q = a.ds->pb_Q;
  const uint32_t* key = a.key[a.passes & 1];
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  for (uint64_t s = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; s < Q; s += stride) {
    const uint32_t p = key[s];
    if (s == 0 || key[s - 1] != p) a.first[p] = (uint32_t)s;
    if (s + 1 == Q || key[s + 1] != p) a.endp[p] = (uint32_t)(s + 1);
  }
}

// Sorted order: the first entry of each chunk (rank a multiple of B among
// its parent's entries) records the chunk's size at its queue position.
__global__ void __launch_bounds__(PB_THREADS) pb_heads_kernel(ParentArgs a) {
  wait_predecessor();
  DevScalars* ds = a.ds;
  const uint64_t Q = ds->pb_Q;
  const uint32_t* key = a.key[a.passes & 1];
  const uint32_t* val = a.val[a.passes & 1];
  const uint32_t B = a.B;
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  for (uint64_t s = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; s < Q; s += stride) {
    const uint32_t p = key[s];
    const uint32_t r = (uint32_t)s - a.first[p];
    if (r % B != 0u) continue;
    const uint32_t i = val[s];
    const uint32_t sz = min(B, a.endp[p] - (uint32_t)s);
    a.hsz[i] = sz;
    if (!a.flush && sz < B) atomicMin(&ds->pb_stop, (unsigned long long)i);
  }
}

// Sorted order, only when a short chunk stops the reservations: entries of
// chunks whose first entry is at or after the stop stay queued.
__global__ void __launch_bounds__(PB_THREADS) pb_mark_kernel(ParentArgs a) {
  wait_predecessor();
  const DevScalars* ds = a.ds;
  const unsigned long long stop = ds->pb_stop;
  if (stop == ~0ull) return;
  const uint64_t Q = ds->pb_Q;
  const uint32_t* key = a.key[a.passes & 1];
  const uint32_t* val = a.val[a.passes & 1];
  const uint32_t B = a.B;
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  for (uint64_t s = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; s < Q; s += stride) {
    const uint32_t f = a.first[key[s]];
    const uint32_t r = (uint32_t)s - f;
    const uint32_t hw = val[f + (r - r % B)];   // queue position of the chunk's first entry
    if (hw >= stop) a.left[val[s]] = 1u;
  }
}

__global__ void __launch_bounds__(PB_THREADS) pb_scan_kernel(ParentArgs a) {
  wait_predecessor();
  __shared__ Pair64 s_scan[33];
  __shared__ uint32_t s_tile;
  __shared__ Pair64 s_prefix;
  DevScalars* ds = a.ds;
  const uint64_t Q = ds->pb_Q;
  const unsigned long long stop = ds->pb_stop;
  const uint32_t B = a.B;
  const uint64_t n_tiles = pb_tiles(Q);
  if (n_tiles == 0) {   // empty window: nothing taken, nothing left
    if (blockIdx.x == 0 && threadIdx.x == 0) {
      ds->pb_npop = ds->pb_nb = ds->pb_R = 0;
      if (a.batch_off && a.off_cap < 1) {
        ds->pb_err = 1u;
        atomicOr(&ds->err, ERR_CAPACITY);
      } else if (a.batch_off) {
        a.batch_off[0] = 0;
      }
      if (a.n_batched_out) *a.n_batched_out = 0;
      if (a.n_batches_out) *a.n_batches_out = 0;
    }
    return;
  }
  const uint32_t n_part = participants(n_tiles);
  if (blockIdx.x >= n_part) return;
  for (;;) {
    if (threadIdx.x == 0) s_tile = claim_tile(&ds->tile_ctr[TS_PARENT]);
    __syncthreads();
    const uint32_t tile = s_tile;
    __syncthreads();
    if (tile >= n_tiles) break;
    const uint64_t i0 = (uint64_t)tile * PB_TILE + (uint64_t)threadIdx.x * PB_ITEMS;
    // a: entries of the taken chunks; b: taken chunks << 32 | entries left
    Pair64 mine{0, 0};
    uint32_t take_head = 0, left = 0, sz[PB_ITEMS];
#pragma unroll
    for (int k = 0; k < PB_ITEMS; ++k) {
      const uint64_t i = i0 + k;
      sz[k] = 0u;
      if (i >= Q) continue;
      sz[k] = a.hsz[i];
      if (a.left[i]) {
        left |= 1u << k;
        mine.b += 1;
      } else if (sz[k] != 0u && i < stop) {
        take_head |= 1u << k;
        mine.a += sz[k];
        mine.b += 1ull << 32;
      }
    }
    Pair64 total;
    const Pair64 excl = block_excl_scan_pair(mine, s_scan, &total);
    if (threadIdx.x < 32) {  // one warp looks back
      const Pair64 pfx = lookback_exclusive(a.ts, tile, total, ds->epoch[TS_PARENT], &ds->err);
      if (threadIdx.x == 0) s_prefix = pfx;
    }
    __syncthreads();
    Pair64 run = s_prefix + excl;
#pragma unroll
    for (int k = 0; k < PB_ITEMS; ++k) {
      const uint64_t i = i0 + k;
      if (take_head & (1u << k)) {
        a.hoff[i] = (uint32_t)run.a;
        const uint64_t b = run.b >> 32;
        if (a.batch_off && b < a.off_cap) a.batch_off[b] = run.a;
        run.a += sz[k];
        run.b += 1ull << 32;
      } else if (left & (1u << k)) {
        a.rem[run.b & 0xFFFFFFFFull] = a.child[i];
        run.b += 1;
      }
    }
    if (tile == n_tiles - 1 && threadIdx.x == PB_THREADS - 1) {
      const unsigned long long npop = run.a, nb = run.b >> 32, R = run.b & 0xFFFFFFFFull;
      ds->pb_npop = npop;
      ds->pb_nb = nb;
      ds->pb_R = R;
      if (a.n_batched_out) *a.n_batched_out = npop;
      if (a.n_batches_out) *a.n_batches_out = nb;
      if (npop > a.cap || (a.batch_off && nb + 1 > a.off_cap)) {
        ds->pb_err = 1u;
        atomicOr(&ds->err, ERR_CAPACITY);
      } else if (a.batch_off) {
        a.batch_off[nb] = npop;
      }
    }
  }
  if (threadIdx.x == 0) retire_cta(ds, TS_PARENT, n_part);
}

__global__ void __launch_bounds__(PB_THREADS) pb_emit_kernel(ParentArgs a) {
  wait_predecessor();
  DevScalars* ds = a.ds;
  const uint64_t Q = ds->pb_Q, head = ds->pb_head;
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  const uint64_t g = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (ds->pb_err) {
    // refused: the admitted Grains go back to WAITING, the tail back
    const uint64_t t0 = ds->pb_old_tail, t1 = head + Q;
    for (uint64_t t = t0 + g; t < t1; t += stride) a.slot[a.queue[t]].phase = WAIT_UNCLAIMED;
    if (g == 0) a.qstate[1] = t0;
    return;
  }
  const unsigned long long stop = ds->pb_stop, npop = ds->pb_npop, R = ds->pb_R;
  const uint32_t* key = a.key[a.passes & 1];
  const uint32_t* val = a.val[a.passes & 1];
  const uint32_t B = a.B;
  // sorted order: a taken chunk's entries are consecutive here and in the
  // output, so the writes to the batches are contiguous
  for (uint64_t s = g; s < Q; s += stride) {
    const uint32_t f = a.first[key[s]];
    const uint32_t r = (uint32_t)s - f, k = r % B;
    const uint32_t hw = val[f + (r - k)];   // queue position of the chunk's first entry
    if (hw >= stop) continue;
    const uint32_t c = a.child[val[s]];
    a.batched[a.hoff[hw] + k] = c;
    a.slot[c].phase = (a.slot[c].phase & ~3u) | PH_INFLIGHT;
  }
  for (uint64_t j = g; j < R; j += stride) a.queue[head + npop + j] = a.rem[j];
  if (g == 0) {
    a.qstate[0] = head + npop;
    ds->stats[5] += ds->pb_bad;
  }
}

void launch_parent(const LaunchCfg& L, const ParentArgs& a) {
  const uint64_t tiles = std::max<uint64_t>(1, ceil_div(a.N, (uint64_t)PB_TILE));
  const int g_elem = (int)std::max<uint64_t>(
      1, std::min<uint64_t>(ceil_div(a.N, (uint64_t)PB_THREADS), (uint64_t)L.grid_pb));
  const int g_tile = (int)std::min<uint64_t>(tiles, (uint64_t)L.grid_pb_sort);
  launch_k(L, K_PB_KEYS, pb_keys_kernel, g_elem, PB_THREADS, 0, a);
  for (int p = 0; p < a.passes; ++p) {
    ParentArgs b = a;
    b.pass = p;
    launch_k(L, K_PB_HIST, pb_hist_kernel, g_tile, PB_THREADS, 0, b);
    launch_k(L, K_PB_ROWSCAN, pb_rowscan_kernel, PB_DIGITS, PB_THREADS, 0, b);
    launch_k(L, K_PB_SORT, pb_sort_kernel, g_tile, PB_THREADS, 0, b);
  }
  launch_k(L, K_PB_BOUNDS, pb_bounds_kernel, g_elem, PB_THREADS, 0, a);
  launch_k(L, K_PB_HEADS, pb_heads_kernel, g_elem, PB_THREADS, 0, a);
  if (!a.flush) launch_k(L, K_PB_MARK, pb_mark_kernel, g_elem, PB_THREADS, 0, a);
  launch_k(L, K_PB_SCAN, pb_scan_kernel, g_tile, PB_THREADS, 0, a);
  launch_k(L, K_PB_EMIT, pb_emit_kernel, g_elem, PB_THREADS, 0, a);
}

const void* kernel_ptr_parent(int which) {
  switch (which) {
    case K_PB_SORT: return (const void*)pb_sort_kernel;
    case K_PB_SCAN: return (const void*)pb_scan_kernel;
    default: return (const void*)pb_heads_kernel;
  }
}

}  // namespace ro
