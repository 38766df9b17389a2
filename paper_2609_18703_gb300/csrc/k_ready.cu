// k_ready.cu — ro_batch_ready kernels (Section 4.3, Eq. 2).
//
// Admission into a per-Call FIFO Ready Queue is an ordered stream compaction
// of the candidate list; elastic reservation then takes whole batches from
// the queue head.  Two passes:
//   ready_count   decides admission.  A candidate list may name a child more
//                 than once; the lowest position wins, through a CAS on the
//                 child's WAITING phase word that keeps the smallest claim.
//                 Counting the transitions out of "unclaimed" gives the exact
//                 number admitted.  The last CTA turns that count into the
//                 reservation (how many leave the queue), checks the output
//                 capacity and advances the queue's head and tail.
//   ready_scatter recomputes the admission flags, ranks them with a
//                 single-pass scan (decoupled look-back) and writes every
//                 admitted child either into the reserved batches (IN-FLIGHT)
//                 or behind the queue's tail (READY).  Queued entries from
//                 earlier calls leave first.
// With the capacity check in the first pass, a call that cannot fit changes
// nothing but the claims, which the second pass then releases.
#include <algorithm>

#include "ro_internal.h"

namespace ro {

__device__ __forceinline__ bool call_ok(const ReadyArgs& a, uint64_t c) {
  return !a.check_call || w_call(a.rec[c].w) == a.call;
}
// A phase word holding claim i (a WAITING child whose first occurrence in
// the candidate list is position i) was claimed by this call.  When other
// Calls' admissions may run at the same time (Call streams), possibly with
// the same candidate list, that holds only for this Call's children; one
// at a time, every other Call's claims are settled before this call starts.
__device__ __forceinline__ bool claimed_here(const ReadyArgs& a, uint64_t c, uint32_t w, uint64_t i) {
  return w == ((uint32_t)i << 2) && (!a.calls_concurrent || call_ok(a, c));
}

__global__ void __launch_bounds__(RB_THREADS) ready_count_kernel(ReadyArgs a) {
  wait_predecessor();
  __shared__ unsigned long long s_red[2][RB_THREADS / 32];
  __shared__ unsigned long long s_scan[33];
  __shared__ uint32_t s_last;
  DevScalars* ds = a.ds;
  ReadyScalars* rs = a.rs;
  unsigned long long kept = 0, bad = 0;
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  for (uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; i < a.n_cand; i += stride) {
    const uint64_t c = a.cand ? (uint64_t)a.cand[i] : i;
    if (c >= a.N) {
      ++bad;
      continue;
    }
    uint32_t w = a.phase[c];
    if ((w & 3u) != PH_WAITING || !call_ok(a, c)) continue;
    if (!a.cand) {
      ++kept;   // ids are distinct: every WAITING child of this Call enters
      continue;
    }
    const uint32_t mine = (uint32_t)i << 2;
    for (;;) {
      if ((w & 3u) != PH_WAITING || (w >> 2) <= (uint32_t)i) break;
      const uint32_t old = atomicCAS(a.phase + c, w, mine);
      if (old == w) {
        if ((w >> 2) == CLAIM_NONE) ++kept;   // first claim of this child
        break;
      }
      w = old;
    }
  }
  // block reduction
  for (int d = 16; d > 0; d >>= 1) {
    kept += __shfl_down_sync(0xffffffffu, kept, d);
    bad += __shfl_down_sync(0xffffffffu, bad, d);
  }
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  if (lane == 0) {
    s_red[0][wid] = kept;
    s_red[1][wid] = bad;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned long long k = 0, b = 0;
    for (int j = 0; j < RB_THREADS / 32; ++j) {
      k += s_red[0][j];
      b += s_red[1][j];
    }
    if (k) atomicAdd(&rs->rb_kept, k);
    if (b) atomicAdd(&rs->rb_bad, b);
    s_last = ticket(&rs->rb_ticket) == gridDim.x - 1;
  }
  __syncthreads();
  if (!s_last) return;
  // last CTA.  Recovery groups (ro_retry) go ahead of the queue's entries,
  // into the slots before the head: each retried Grain was taken out of this
  // queue once, so there are at least as many such slots.
  const unsigned long long nr = a.qstate[2], h0 = a.qstate[0];
  const unsigned long long mv = nr < h0 ? nr : h0;
  for (unsigned long long j = threadIdx.x; j < mv; j += RB_THREADS) a.queue[h0 - mv + j] = a.rq[j];
  if (mv != nr && threadIdx.x == 0) atomicOr(&ds->err, ERR_INVAL);   // cannot happen
  __syncthreads();
  // Queued Grains that a GroupFailure has sealed since they were queued
  // leave the queue now, undispatched (Section 4.4): stable in-place
  // compaction of the queue window (fewer than one batch is usually left over).
  const unsigned long long head = h0 - mv, tail0 = a.qstate[1];
  unsigned long long tail = head;
  for (unsigned long long base = head; base < tail0; base += RB_THREADS) {
    const unsigned long long i = base + threadIdx.x;
    uint32_t c = 0;
    bool live = false;
    if (i < tail0) {
      c = a.queue[i];
      live = (a.phase[c] & 3u) == PH_READY;
    }
    unsigned long long total;
    const unsigned long long pos = block_excl_scan((unsigned long long)live, s_scan, &total);
    if (live) a.queue[tail + pos] = c;   // never ahead of an entry not yet read
    tail += total;
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    {
      // plan the reservation
      if (tail0 != tail) atomicAdd(&ds->stats[10], tail0 - tail);   // Calls may run at once
      a.qstate[0] = head;
      a.qstate[1] = tail;
      a.qstate[2] = 0;
      const unsigned long long K = ld_relaxed_u64(&rs->rb_kept);
      const unsigned long long L = tail - head, T = L + K;
      // parent-bound reservation takes nothing here: everything admitted is
      // queued and the window [head, head + T) goes to launch_parent
      const unsigned long long npop =
          a.parent_bound ? 0ull : a.flush ? T : (T / a.batch_size) * a.batch_size;
      if (a.parent_bound) {
        ds->pb_Q = T;
        ds->pb_head = head;
        ds->pb_old_tail = tail;
        ds->pb_stop = ~0ull;
        ds->pb_bad = ld_relaxed_u64(&rs->rb_bad);
        ds->pb_err = 0u;
      }
      rs->rb_npop = npop;
      rs->rb_n_batches = (npop + a.batch_size - 1) / a.batch_size;
      if (a.n_batched_out) *a.n_batched_out = npop;
      if (npop > a.cap) {
        rs->rb_err = 1u;
        atomicOr(&ds->err, ERR_CAPACITY);
      } else {
        rs->rb_err = 0u;
        rs->rb_L = L;
        rs->rb_k = K;
        rs->rb_head = head;
        rs->rb_tail = tail;
        a.qstate[0] = head + npop;
        a.qstate[1] = tail + K;
        if (!a.parent_bound) atomicAdd(&ds->stats[5], ld_relaxed_u64(&rs->rb_bad));
      }
      rs->rb_kept = 0;
      rs->rb_bad = 0;
      rs->rb_ticket = 0u;
    }
  }
}

__global__ void __launch_bounds__(RB_THREADS) ready_scatter_kernel(ReadyArgs a) {
  wait_predecessor();
  __shared__ unsigned long long s_scan[33];
  __shared__ uint32_t s_tile;
  __shared__ unsigned long long s_prefix;
  DevScalars* ds = a.ds;
  ReadyScalars* rs = a.rs;
  const bool failed = rs->rb_err != 0u;
  const unsigned long long L = rs->rb_L, npop = rs->rb_npop, head = rs->rb_head;

  if (failed) {
    // release the claims taken by the first pass; nothing else changes
    if (a.cand) {
      const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
      for (uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; i < a.n_cand; i += stride) {
        const uint64_t c = a.cand[i];
        if (c < a.N && claimed_here(a, c, a.phase[c], i)) a.phase[c] = WAIT_UNCLAIMED;
      }
    }
    return;   // no tile counter was touched
  }

  const uint64_t TILE = (uint64_t)RB_THREADS * RB_ITEMS;
  const uint64_t n_tiles = ceil_div(a.n_cand, TILE);
  const unsigned long long n_old = L < npop ? L : npop;
  const uint64_t units = n_tiles > ceil_div(n_old, TILE) ? n_tiles : ceil_div(n_old, TILE);
  const uint32_t n_part = participants(units);
  if (blockIdx.x >= n_part) return;

  // entries queued by earlier calls leave first
  {
    const uint64_t stride = (uint64_t)n_part * blockDim.x;
    for (uint64_t j = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; j < n_old; j += stride) {
      const uint32_t c = a.queue[head + j];
      a.batched[j] = c;
      a.phase[c] = (a.phase[c] & ~3u) | PH_INFLIGHT;
    }
  }

  for (;;) {
    if (threadIdx.x == 0) s_tile = claim_tile(&rs->tile_ctr);
    __syncthreads();
    const uint32_t tile = s_tile;
    __syncthreads();
    if (tile >= n_tiles) break;
    const uint64_t i0 = tile * TILE + (uint64_t)threadIdx.x * RB_ITEMS;
    uint32_t cs[RB_ITEMS];
    uint32_t flags = 0;
    unsigned long long cnt = 0;
#pragma unroll
    for (int k = 0; k < RB_ITEMS; ++k) {
      const uint64_t i = i0 + k;
      cs[k] = 0;
      if (i >= a.n_cand) continue;
      const uint64_t c = a.cand ? (uint64_t)a.cand[i] : i;
      if (c >= a.N) continue;
      const uint32_t w = a.phase[c];
      const bool keep = a.cand ? claimed_here(a, c, w, i) : (w == WAIT_UNCLAIMED && call_ok(a, c));
      if (keep) {
        flags |= 1u << k;
        cs[k] = (uint32_t)c;
        ++cnt;
      }
    }
    unsigned long long total;
    unsigned long long excl = block_excl_scan(cnt, s_scan, &total);
    if (threadIdx.x < 32) {  // one warp looks back
      const auto pfx = lookback_exclusive(a.ts, tile, total, rs->epoch, &ds->err);
      if (threadIdx.x == 0) s_prefix = pfx;
    }
    __syncthreads();
    unsigned long long rank = s_prefix + excl;
#pragma unroll
    for (int k = 0; k < RB_ITEMS; ++k) {
      if (!(flags & (1u << k))) continue;
      const uint32_t c = cs[k];
      const unsigned long long j = L + rank;   // position in the logical queue
      if (j < npop) {
        a.batched[j] = c;
        a.phase[c] = ph_make(PH_INFLIGHT, 0u);
      } else {
        a.queue[head + j] = c;
        a.phase[c] = ph_make(PH_READY, 0u);
      }
      ++rank;
    }
  }
  if (threadIdx.x == 0 && ticket(&rs->exit_ctr) == n_part - 1) {
    rs->tile_ctr = 0u;
    rs->exit_ctr = 0u;
    rs->epoch += 1ull;
  }
}

void launch_ready(const LaunchCfg& L, const ReadyArgs& a) {
  const uint64_t per = (uint64_t)RB_THREADS;
  const int grid_count =
      (int)std::max<uint64_t>(1, std::min<uint64_t>(ceil_div(a.n_cand, per), (uint64_t)L.grid_rb));
  launch_k(L, K_RB_COUNT, ready_count_kernel, grid_count, RB_THREADS, 0, a);
  // one CTA per tile of candidates; CTAs past them only help move the
  // entries earlier calls queued (a grid-stride loop), for which one per SM
  // is plenty
  const uint64_t tiles = ceil_div(a.n_cand, (uint64_t)RB_THREADS * RB_ITEMS);
  const int grid_scatter = (int)std::min<uint64_t>(
      (uint64_t)L.grid_rb, std::max<uint64_t>(tiles, std::max(1, L.grid_rb / 8)));
  launch_k(L, K_RB_SCATTER, ready_scatter_kernel, grid_scatter, RB_THREADS, 0, a);
}

const void* kernel_ptr_ready(int which) {
  return which == K_RB_COUNT ? (const void*)ready_count_kernel : (const void*)ready_scatter_kernel;
}

}  // namespace ro
