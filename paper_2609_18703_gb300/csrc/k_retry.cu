// k_retry.cu — ro_retry kernels (Section 4.4: a failed physical attempt is
// retried at a higher generation; Eq. 2's IN-FLIGHT -> READY edge; Section
// 4.3: recovery queues).
//
// retry_claim    entries naming an IN-FLIGHT Grain of the Call claim it;
//                the lowest list position wins (a max over the complemented
//                position, kept in the record's len field, which is unused
//                while a Grain is in flight).
// retry_scatter  the winners, ranked in list order by a single-pass scan
//                (decoupled look-back), go back to READY with generation + 1
//                and are appended to the Call's recovery queue as one group;
//                each clears its claim.  The next ro_batch_ready places the
//                recovery groups ahead of the Ready Queue's entries.
#include <algorithm>

#include "ro_internal.h"

namespace ro {

// Grain c is a target: IN-FLIGHT and of the Call (from its slot v, read
// whole: phase word, len and w share one sector).
__device__ __forceinline__ bool retry_target(const RetryArgs& a, const Slot& v) {
  if ((v.phase & 3u) != PH_INFLIGHT) return false;
  return !a.check_call || w_call(v.w) == a.call;
}
__device__ __forceinline__ Slot load_slot(const Slot* p) {
  const ulonglong2 v = __ldcg(reinterpret_cast<const ulonglong2*>(p));
  Slot s;
  s.phase = (uint32_t)v.x;
  s.len = (uint32_t)(v.x >> 32);
  s.w = v.y;
  return s;
}

__global__ void __launch_bounds__(RT_THREADS) retry_claim_kernel(RetryArgs a) {
  wait_predecessor();
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  for (uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; i < a.n; i += stride) {
    const uint64_t c = a.children[i];
    if (c < a.N && retry_target(a, load_slot(a.slot + c))) atomicMax(&a.slot[c].len, ~(uint32_t)i);
  }
}

__global__ void __launch_bounds__(RT_THREADS) retry_scatter_kernel(RetryArgs a) {
  wait_predecessor();
  __shared__ unsigned long long s_scan[33];
  __shared__ uint32_t s_tile;
  __shared__ unsigned long long s_prefix;
  DevScalars* ds = a.ds;
  const uint64_t TILE = (uint64_t)RT_THREADS * RT_ITEMS;
  const uint64_t n_tiles = ceil_div(a.n, TILE);
  const unsigned long long rlen = a.qstate[2];
  if (n_tiles == 0) return;
  const uint32_t n_part = participants(n_tiles);
  if (blockIdx.x >= n_part) return;
  for (;;) {
    if (threadIdx.x == 0) s_tile = claim_tile(&ds->tile_ctr[TS_RETRY]);
    __syncthreads();
    const uint32_t tile = s_tile;
    __syncthreads();
    if (tile >= n_tiles) break;
    const uint64_t i0 = tile * TILE + (uint64_t)threadIdx.x * RT_ITEMS;
    // the group's entries, then their slots, every load in flight at once
    uint32_t cs[RT_ITEMS], phs[RT_ITEMS];
#pragma unroll
    for (int k = 0; k < RT_ITEMS; ++k) cs[k] = i0 + k < a.n ? a.children[i0 + k] : 0u;
    uint32_t flags = 0;
#pragma unroll
    for (int k = 0; k < RT_ITEMS; ++k) {
      phs[k] = 0;
      if (i0 + k < a.n && cs[k] < a.N) {
        const Slot v = load_slot(a.slot + cs[k]);
        // the winner still sees its own claim; a later entry for the same
        // Grain sees another claim or the cleared one
        if (retry_target(a, v) && v.len == ~(uint32_t)(i0 + k)) {
          flags |= 1u << k;
          phs[k] = v.phase;
        }
      }
    }
    const unsigned long long cnt = __popc(flags);
    unsigned long long total;
    const unsigned long long excl = block_excl_scan(cnt, s_scan, &total);
    if (threadIdx.x < 32) {  // one warp looks back
      const auto pfx = lookback_exclusive(a.ts, tile, total, ds->epoch[TS_RETRY], &ds->err);
      if (threadIdx.x == 0) s_prefix = pfx;
    }
    __syncthreads();
    unsigned long long rank = s_prefix + excl;
#pragma unroll
    for (int k = 0; k < RT_ITEMS; ++k) {
      if (!(flags & (1u << k))) continue;
      const uint32_t c = cs[k];
      a.rq[rlen + rank] = c;
      a.slot[c].len = 0u;
      a.slot[c].phase = ph_make(PH_READY, (phs[k] >> 2) + 1u);
      ++rank;
    }
    if (tile == n_tiles - 1 && threadIdx.x == RT_THREADS - 1) {
      const unsigned long long done = rank;   // winners over the whole list
      a.qstate[2] = rlen + done;
      ds->stats[11] += done;
      ds->stats[12] += a.n - done;
      ds->rt_done = done;
    }
  }
  if (threadIdx.x == 0) retire_cta(ds, TS_RETRY, n_part);
}

void launch_retry(const LaunchCfg& L, const RetryArgs& a) {
  const uint64_t tiles = ceil_div(a.n, (uint64_t)RT_THREADS * RT_ITEMS);
  const int g1 = (int)std::max<uint64_t>(1, std::min<uint64_t>(ceil_div(a.n, RT_THREADS), (uint64_t)L.grid_retry));
  launch_k(L, K_RT_CLAIM, retry_claim_kernel, g1, RT_THREADS, 0, a);
  const int g2 = (int)std::max<uint64_t>(1, std::min<uint64_t>(tiles, (uint64_t)L.grid_retry));
  launch_k(L, K_RT_SCATTER, retry_scatter_kernel, g2, RT_THREADS, 0, a);
}

const void* kernel_ptr_retry(int which) {
  return which == K_RT_CLAIM ? (const void*)retry_claim_kernel : (const void*)retry_scatter_kernel;
}

}  // namespace ro
