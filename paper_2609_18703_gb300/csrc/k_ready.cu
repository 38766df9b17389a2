// k_ready.cu — ro_batch_ready kernels (Section 4.3, Eq. 2).
//
// Admission into a per-Call FIFO Ready Queue is an ordered stream compaction
// of the candidate list; elastic reservation then takes whole batches from
// the queue head.  A candidate list may name a child more than once; the
// lowest position wins, through a CAS on the child's WAITING phase word that
// keeps the smallest claim.  Lists of up to a few thousand tiles of 2,048
// candidates take one kernel:
//   ready_fused   cooperative launch, one CTA per tile plus one for the
//                 queue window: claims and per-tile admitted counts, a grid
//                 barrier (and, only when some child was named twice, a
//                 recount and a second one), then every CTA knows its tile's
//                 prefix and the reservation and writes its children into the
//                 reserved batches (IN-FLIGHT) or behind the queue's tail
//                 (READY); the window's CTA compacts the window meanwhile,
//                 and the entries earlier calls queued leave first, a slice
//                 per CTA.  ready_fused_calls runs several Calls' admissions
//                 from one candidate list in one such grid.
// Longer lists (and every list with RO_ADMIT_TWO_PASS set) take two:
//   ready_count   decides admission.  Counting the claims' transitions out of
//                 "unclaimed" gives the exact number admitted.  The last CTA
//                 compacts the window, turns that count into the reservation
//                 (how many leave the queue), checks the output capacity and
//                 advances the queue's head and tail.
//   ready_scatter recomputes the admission flags, ranks them with a
//                 single-pass scan (decoupled look-back) and writes as above.
// A call that cannot fit changes nothing but the claims, which are then
// released, and the window's compaction (sealed entries would leave anyway).
#include <algorithm>

#include "ro_internal.h"

namespace ro {

// One thread's group of RB_ITEMS candidate positions of a tile (striped:
// position base + k * RB_THREADS + thread, so that each load instruction of
// a warp reads consecutive positions): the child each names and that
// child's phase word and Call, loaded so that every load of the group is in
// flight at once (first the candidates, then the slots; one 16-byte slot
// holds both fields).
struct CandGroup {
  uint32_t c[RB_ITEMS];
  uint32_t ph[RB_ITEMS];
  uint32_t call[RB_ITEMS];
  uint32_t in_range;   // bit k: position cand_pos(base, k) < n_cand
  uint32_t valid;      // bit k: in range and names a child of the expansion
};
__device__ __forceinline__ uint64_t cand_pos(uint64_t base, int k) {
  return base + (uint64_t)k * RB_THREADS + threadIdx.x;
}
__device__ __forceinline__ void load_group(const ReadyArgs& a, uint64_t base, CandGroup& g) {
  g.in_range = 0u;
  g.valid = 0u;
#pragma unroll
  for (int k = 0; k < RB_ITEMS; ++k) {
    const uint64_t i = cand_pos(base, k);
    const bool in = i < a.n_cand;
    g.c[k] = in ? (a.cand ? a.cand[i] : (uint32_t)i) : 0u;
    if (in) g.in_range |= 1u << k;
  }
#pragma unroll
  for (int k = 0; k < RB_ITEMS; ++k) {
    const bool ok = ((g.in_range >> k) & 1u) && g.c[k] < a.N;
    if (ok) g.valid |= 1u << k;
    g.ph[k] = WAIT_UNCLAIMED;
    g.call[k] = 0u;
    if (ok) {
      const ulonglong2 v = __ldcg(reinterpret_cast<const ulonglong2*>(a.slot + g.c[k]));
      g.ph[k] = (uint32_t)v.x;
      g.call[k] = w_call(v.y);
    }
  }
}
__device__ __forceinline__ bool call_ok(const ReadyArgs& a, uint32_t call) {
  return !a.check_call || call == a.call;
}
// A phase word holding claim i (a WAITING child whose first occurrence in
// the candidate list is position i) was claimed by this call.  When other
// Calls' admissions may run at the same time (Call streams), possibly with
// the same candidate list, that holds only for this Call's children; one
// at a time, every other Call's claims are settled before this call starts.
__device__ __forceinline__ bool claimed_here(const ReadyArgs& a, uint32_t call, uint32_t w, uint64_t i) {
  return w == ((uint32_t)i << 2) && (!a.calls_concurrent || call_ok(a, call));
}
// Whether candidate k of a group enters the queue, once every claim is settled.
__device__ __forceinline__ bool admitted(const ReadyArgs& a, const CandGroup& g, int k, uint64_t i) {
  if (!((g.valid >> k) & 1u)) return false;
  return a.cand ? claimed_here(a, g.call[k], g.ph[k], i)
                : (g.ph[k] == WAIT_UNCLAIMED && call_ok(a, g.call[k]));
}

// Claims of a group's eligible candidates: the lowest position keeps the
// child (a CAS that keeps the smallest claim in its WAITING phase word).
// First attempts are all in flight together, then the (rare) ones that met
// another claim retry.  Returns the number of first claims (transitions out
// of "unclaimed"): summed over the list, the number of distinct children
// admitted.
__device__ __forceinline__ uint32_t claim_group(const ReadyArgs& a, uint64_t base, const CandGroup& g,
                                                uint32_t elig) {
  uint32_t old[RB_ITEMS], firsts = 0;
#pragma unroll
  for (int k = 0; k < RB_ITEMS; ++k) {
    old[k] = g.ph[k];
    const uint32_t i = (uint32_t)cand_pos(base, k);
    if (((elig >> k) & 1u) && (g.ph[k] >> 2) > i)
      old[k] = atomicCAS(&a.slot[g.c[k]].phase, g.ph[k], i << 2);
    else
      elig &= ~(1u << k);
  }
#pragma unroll
  for (int k = 0; k < RB_ITEMS; ++k) {
    if (!((elig >> k) & 1u)) continue;
    const uint32_t i = (uint32_t)cand_pos(base, k), mine = i << 2;
    uint32_t w = g.ph[k], o = old[k];
    bool won = o == w;
    while (!won) {   // another claim got there first
      w = o;
      if ((w & 3u) != PH_WAITING || (w >> 2) <= i) break;
      o = atomicCAS(&a.slot[g.c[k]].phase, w, mine);
      won = o == w;
    }
    if (won && (w >> 2) == CLAIM_NONE) ++firsts;   // first claim of this child
  }
  return firsts;
}

// The same claims for the one-pass admission: *won = the candidates whose
// claim this thread took (they stand unless a child is named twice).
// Returns whether any claim met another one (a repeat somewhere in the list).
__device__ __forceinline__ bool claim_group_won(const ReadyArgs& a, uint64_t base, const CandGroup& g,
                                                uint32_t elig, uint32_t* won) {
  uint32_t old[RB_ITEMS], w = 0u;
  bool conflict = false;
#pragma unroll
  for (int k = 0; k < RB_ITEMS; ++k) {
    old[k] = g.ph[k];
    if (!((elig >> k) & 1u)) continue;
    const uint32_t i = (uint32_t)cand_pos(base, k);
    if ((g.ph[k] >> 2) != CLAIM_NONE) conflict = true;   // claimed before this attempt
    if ((g.ph[k] >> 2) > i) old[k] = atomicCAS(&a.slot[g.c[k]].phase, g.ph[k], i << 2);
  }
#pragma unroll
  for (int k = 0; k < RB_ITEMS; ++k) {
    if (!((elig >> k) & 1u)) continue;
    const uint32_t i = (uint32_t)cand_pos(base, k), mine = i << 2;
    if ((g.ph[k] >> 2) <= i) continue;   // a lower position holds it
    uint32_t cur = g.ph[k], o = old[k];
    bool ok = o == cur;
    while (!ok) {   // another claim got there first
      conflict = true;
      cur = o;
      if ((cur & 3u) != PH_WAITING || (cur >> 2) <= i) break;
      o = atomicCAS(&a.slot[g.c[k]].phase, cur, mine);
      ok = o == cur;
    }
    if (ok) w |= 1u << k;
  }
  *won = w;
  return conflict;
}

// A tile's admitted and bad counts, summed over the CTA, into the per-tile
// arrays (the look-back buffers' value arrays) for the other CTAs.
__device__ __forceinline__ void publish_counts(const ReadyArgs& a, uint32_t tile, uint32_t flags, const CandGroup& g,
                                               unsigned long long (*s_red)[RB_THREADS / 32]) {
  unsigned long long kept = __popc(flags), bad = __popc(g.in_range & ~g.valid);
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
    a.ts.agg[tile] = k;
    a.ts.inc[tile] = b;
  }
  __syncthreads();
}

// Eligible candidates of a group: naming a WAITING child of this Call.
__device__ __forceinline__ uint32_t eligible(const ReadyArgs& a, const CandGroup& g) {
  uint32_t elig = 0u;
#pragma unroll
  for (int k = 0; k < RB_ITEMS; ++k)
    if (((g.valid >> k) & 1u) && (g.ph[k] & 3u) == PH_WAITING && call_ok(a, g.call[k])) elig |= 1u << k;
  return elig;
}

// Ranks of a tile's flagged candidates in position order (striped layout):
// rowpfx[k] = flagged positions before this thread's item k in the tile.
// Returns the tile's total.  Row k, warp w holds positions k * RB_THREADS +
// 32 w + lane, so the order is (row, warp, lane).
__device__ __forceinline__ uint32_t rank_rows(uint32_t flags, uint32_t* s_rows, uint32_t (&rowpfx)[RB_ITEMS]) {
  constexpr int NW = RB_THREADS / 32, NE = RB_ITEMS * NW;
  static_assert(NE == 64, "two row-warp counts per lane");
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const uint32_t lt = (1u << lane) - 1u;
  uint32_t bal[RB_ITEMS];
#pragma unroll
  for (int k = 0; k < RB_ITEMS; ++k) {
    bal[k] = __ballot_sync(0xffffffffu, (flags >> k) & 1u);
    if (lane == 0) s_rows[k * NW + wid] = __popc(bal[k]);
  }
  __syncthreads();
  if (wid == 0) {   // exclusive scan of the 64 counts in (row, warp) order
    const uint32_t x0 = s_rows[2 * lane], x1 = s_rows[2 * lane + 1];
    uint32_t inc = x0 + x1;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      const uint32_t u = __shfl_up_sync(0xffffffffu, inc, d);
      if (lane >= d) inc += u;
    }
    const uint32_t ex = inc - x0 - x1;
    s_rows[2 * lane] = ex;
    s_rows[2 * lane + 1] = ex + x0;
    s_rows[NE] = __shfl_sync(0xffffffffu, inc, 31);
  }
  __syncthreads();
#pragma unroll
  for (int k = 0; k < RB_ITEMS; ++k) rowpfx[k] = s_rows[k * NW + wid] + __popc(bal[k] & lt);
  const uint32_t total = s_rows[NE];
  __syncthreads();   // s_rows is reused by the next tile
  return total;
}

// The queue window, by the whole CTA.  Recovery groups (ro_retry) go ahead
// of the queue's entries, into the slots before the head: each retried
// Grain was taken out of this queue once, so there are at least as many such
// slots.  Queued Grains that a GroupFailure has sealed since they were
// queued leave the queue now, undispatched (Section 4.4): stable in-place
// compaction of the window, 2,048 entries at a time (fewer than one batch is
// usually left over).  Returns the window's head, its tail after and before.
__device__ void compact_window(const ReadyArgs& a, unsigned long long* s_scan, unsigned long long* head_out,
                               unsigned long long* tail_out, unsigned long long* tail0_out) {
  const uint64_t TILE = (uint64_t)RB_THREADS * RB_ITEMS;
  const unsigned long long nr = a.qstate[2], h0 = a.qstate[0];
  const unsigned long long mv = nr < h0 ? nr : h0;
  for (unsigned long long j = threadIdx.x; j < mv; j += RB_THREADS) a.queue[h0 - mv + j] = a.rq[j];
  if (mv != nr && threadIdx.x == 0) atomicOr(&a.ds->err, ERR_INVAL);   // cannot happen
  __syncthreads();
  const unsigned long long head = h0 - mv, tail0 = a.qstate[1];
  unsigned long long tail = head;
  for (unsigned long long base = head; base < tail0; base += TILE) {
    const unsigned long long i0 = base + (unsigned long long)threadIdx.x * RB_ITEMS;
    uint32_t cq[RB_ITEMS];
    uint32_t live = 0u;
#pragma unroll
    for (int k = 0; k < RB_ITEMS; ++k) cq[k] = i0 + k < tail0 ? a.queue[i0 + k] : 0u;
#pragma unroll
    for (int k = 0; k < RB_ITEMS; ++k)
      if (i0 + k < tail0 && (__ldcg(&a.slot[cq[k]].phase) & 3u) == PH_READY) live |= 1u << k;
    unsigned long long total;
    unsigned long long pos = block_excl_scan((unsigned long long)__popc(live), s_scan, &total);
    // every entry of this window was read before the scan's barrier, and
    // none is written ahead of its own position
#pragma unroll
    for (int k = 0; k < RB_ITEMS; ++k)
      if ((live >> k) & 1u) a.queue[tail + pos++] = cq[k];
    tail += total;
    __syncthreads();
  }
  *head_out = head;
  *tail_out = tail;
  *tail0_out = tail0;
}

// The reservation (one thread): the window [head, tail) (tail0 before
// compaction) plus K admitted, bad candidates counted.  Elastic: whole
// batches leave (all with flush); parent-bound: nothing here, the window
// goes to launch_parent.  A reservation larger than the output capacity
// fails the call (rb_err): the queue keeps its (compacted) window and the
// claims are released (by the scatter pass, or in the one-pass admission
// by the CTAs that took them).
__device__ void plan_reservation(const ReadyArgs& a, unsigned long long head, unsigned long long tail,
                                 unsigned long long tail0, unsigned long long K, unsigned long long bad) {
  DevScalars* ds = a.ds;
  ReadyScalars* rs = a.rs;
  if (tail0 != tail) atomicAdd(&ds->stats[10], tail0 - tail);   // Calls may run at once
  a.qstate[0] = head;
  a.qstate[1] = tail;
  a.qstate[2] = 0;
  const unsigned long long L = tail - head, T = L + K;
  const unsigned long long npop =
      a.parent_bound ? 0ull : a.flush ? T : (T / a.batch_size) * a.batch_size;
  if (a.parent_bound) {
    ds->pb_Q = T;
    ds->pb_head = head;
    ds->pb_old_tail = tail;
    ds->pb_stop = ~0ull;
    ds->pb_bad = bad;
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
    if (!a.parent_bound) atomicAdd(&ds->stats[5], bad);
  }
}

__global__ void __launch_bounds__(RB_THREADS) ready_count_kernel(ReadyArgs a) {
  wait_predecessor();
  __shared__ unsigned long long s_red[2][RB_THREADS / 32];
  __shared__ unsigned long long s_scan[33];
  __shared__ uint32_t s_last;
  DevScalars* ds = a.ds;
  ReadyScalars* rs = a.rs;
  unsigned long long kept = 0, bad = 0;
  const uint64_t TILE = (uint64_t)RB_THREADS * RB_ITEMS;
  for (uint64_t base = (uint64_t)blockIdx.x * TILE; base < a.n_cand; base += (uint64_t)gridDim.x * TILE) {
    CandGroup g;
    load_group(a, base, g);
    bad += __popc(g.in_range & ~g.valid);
    const uint32_t elig = eligible(a, g);
    if (!a.cand) {   // ids are distinct: every WAITING child of this Call enters
      kept += __popc(elig);
      continue;
    }
    kept += claim_group(a, base, g, elig);
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
  // last CTA: the queue window, then the reservation
  unsigned long long head, tail, tail0;
  compact_window(a, s_scan, &head, &tail, &tail0);
  if (threadIdx.x == 0)
    plan_reservation(a, head, tail, tail0, ld_relaxed_u64(&rs->rb_kept), ld_relaxed_u64(&rs->rb_bad));
  if (threadIdx.x == 0) {
    rs->rb_kept = 0;
    rs->rb_bad = 0;
    rs->rb_ticket = 0u;
  }
}

__global__ void __launch_bounds__(RB_THREADS) ready_scatter_kernel(ReadyArgs a) {
  wait_predecessor();
  __shared__ uint32_t s_rows[RB_ITEMS * (RB_THREADS / 32) + 1];
  __shared__ uint32_t s_tile;
  __shared__ unsigned long long s_prefix;
  DevScalars* ds = a.ds;
  ReadyScalars* rs = a.rs;
  const bool failed = rs->rb_err != 0u;
  const unsigned long long L = rs->rb_L, npop = rs->rb_npop, head = rs->rb_head;

  if (failed) {
    // release the claims taken by the first pass; nothing else changes
    if (a.cand) {
      const uint64_t TILE = (uint64_t)RB_THREADS * RB_ITEMS;
      for (uint64_t base = (uint64_t)blockIdx.x * TILE; base < a.n_cand; base += (uint64_t)gridDim.x * TILE) {
        CandGroup g;
        load_group(a, base, g);
#pragma unroll
        for (int k = 0; k < RB_ITEMS; ++k)
          if (admitted(a, g, k, cand_pos(base, k))) a.slot[g.c[k]].phase = WAIT_UNCLAIMED;
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
      a.slot[c].phase = (a.slot[c].phase & ~3u) | PH_INFLIGHT;
    }
  }

  // with at least as many CTAs as tiles, each CTA claims once
  const bool one_claim = n_tiles <= n_part;
  for (;;) {
    if (threadIdx.x == 0) s_tile = claim_tile(&rs->tile_ctr);
    __syncthreads();
    const uint32_t tile = s_tile;
    __syncthreads();
    if (tile >= n_tiles) break;
    const uint64_t base = tile * TILE;
    CandGroup g;
    load_group(a, base, g);
    uint32_t rowpfx[RB_ITEMS];
    uint32_t flags = 0;
#pragma unroll
    for (int k = 0; k < RB_ITEMS; ++k)
      if (admitted(a, g, k, cand_pos(base, k))) flags |= 1u << k;
    const uint32_t total = rank_rows(flags, s_rows, rowpfx);
    if (threadIdx.x < 32) {  // one warp looks back
      const auto pfx = lookback_exclusive(a.ts, tile, (unsigned long long)total, rs->epoch, &ds->err);
      if (threadIdx.x == 0) s_prefix = pfx;
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < RB_ITEMS; ++k) {
      if (!(flags & (1u << k))) continue;
      const uint32_t c = g.c[k];
      const unsigned long long j = L + s_prefix + rowpfx[k];   // position in the logical queue
      if (j < npop) {
        a.batched[j] = c;
        a.slot[c].phase = ph_make(PH_INFLIGHT, 0u);
      } else {
        a.queue[head + j] = c;
        a.slot[c].phase = ph_make(PH_READY, 0u);
      }
    }
    if (one_claim) break;
  }
  if (threadIdx.x == 0 && ticket(&rs->exit_ctr) == n_part - 1) {
    rs->tile_ctr = 0u;
    rs->exit_ctr = 0u;
    rs->epoch += 1ull;
  }
}


// ---- one-pass admission ---------------------------------------------------------------
// For candidate lists of at most a few thousand tiles: CTAs 0 .. T-1 take one
// tile each, CTA T the queue window.  The launch is cooperative (every CTA
// resident at once), so the CTAs can meet at grid barriers: after the claims
// (explicit lists only) and after the per-tile counts.  Then every CTA knows
// its tile's prefix, the number admitted, the window's live length and so
// the reservation, and writes; no second launch and no look-back.

// The one-pass admission of Call a by CTA b of the Call's T + 1 (T tiles,
// then the window).  gs holds the grid's barrier (one per launch, the first
// Call's); every CTA of the grid meets at the same barriers.
__device__ __forceinline__ void fused_admit(const ReadyArgs a, uint32_t T, uint32_t b, ReadyScalars* gs) {
  __shared__ unsigned long long s_scan[33];
  __shared__ uint32_t s_rows[RB_ITEMS * (RB_THREADS / 32) + 1];
  __shared__ unsigned long long s_red[2][RB_THREADS / 32];
  __shared__ unsigned long long s_tot[5];   // prefix of this tile, admitted, bad, window length, head
  DevScalars* ds = a.ds;
  ReadyScalars* rs = a.rs;
  const bool window = b == T;
  const uint64_t base = (uint64_t)b * RB_THREADS * RB_ITEMS;
  // per-tile counts (admitted, bad), in the look-back buffers' value arrays
  unsigned long long* cnt_kept = a.ts.agg;
  unsigned long long* cnt_bad = a.ts.inc;
  CandGroup g;
  uint32_t flags = 0u, elig = 0u;
  unsigned long long head = 0, tail = 0, tail0 = 0;

  // The candidate list is the caller's input: warm L2 with this CTA's
  // lines while the previous kernel drains, then wait for it (lineage state
  // may still change until then), and let the next kernel launch.
  if (!window && a.cand && threadIdx.x < RB_THREADS * RB_ITEMS / 32) {   // one 128-byte line each
    const uint64_t i = base + (uint64_t)threadIdx.x * 32;
    if (i < a.n_cand) asm volatile("prefetch.global.L2 [%0];" ::"l"(a.cand + i));
  }
  wait_predecessor();
  allow_successor();
  // the barrier generation, read with the first loads (no barrier of this
  // launch completes before this CTA arrives)
  const uint32_t gen0 = __ldcg(&gs->bar_gen) & ~BAR_FLAG;
  bool conflict = false;

  // A: candidates, slots and claims; the window is compacted meanwhile.  A
  // claim that met another one (a child named twice) is reported at the
  // barrier; without any, every claim taken stands and the tile counts
  // below are final.
  if (!window) {
    load_group(a, base, g);
    elig = eligible(a, g);
    if (a.cand) {
      conflict = __syncthreads_or(claim_group_won(a, base, g, elig, &flags)) != 0;
    } else {
      flags = elig;   // ids are distinct
    }
    publish_counts(a, b, flags, g, s_red);
  } else {
    compact_window(a, s_scan, &head, &tail, &tail0);
    if (threadIdx.x == 0) {
      rs->rb_head = head;   // the window, for the other CTAs
      rs->rb_L = tail - head;
    }
  }
  const bool repeats = grid_barrier(gs, (gen0 + 1u) & ~BAR_FLAG, &ds->err, conflict);

  // B (repeats only): with every claim settled, a candidate is admitted iff
  // its child holds its claim; the tile counts again
  if (repeats) {
    if (!window) {
      uint32_t ph[RB_ITEMS];
#pragma unroll
      for (int k = 0; k < RB_ITEMS; ++k)
        ph[k] = ((elig >> k) & 1u) ? __ldcg(&a.slot[g.c[k]].phase) : 0u;
      flags = 0u;
#pragma unroll
      for (int k = 0; k < RB_ITEMS; ++k)
        if (((elig >> k) & 1u) && ph[k] == ((uint32_t)cand_pos(base, k) << 2)) flags |= 1u << k;
      publish_counts(a, b, flags, g, s_red);
    }
    grid_barrier(gs, (gen0 + 2u) & ~BAR_FLAG, &ds->err);
  }

  // C: prefix of this tile, number admitted and bad, and the window (one
  // warp; all its loads in flight together)
  if (threadIdx.x < 32) {
    unsigned long long pre = 0, K = 0, bad = 0, wL = 0, wH = 0;
    if (threadIdx.x == 0 && !window) {
      wL = __ldcg(&rs->rb_L);
      wH = __ldcg(&rs->rb_head);
    }
    for (uint32_t t = threadIdx.x; t < T; t += 32) {
      const unsigned long long k = __ldcg(cnt_kept + t);
      K += k;
      if (t < b) pre += k;
      bad += __ldcg(cnt_bad + t);
    }
    for (int d = 16; d > 0; d >>= 1) {
      pre += __shfl_down_sync(0xffffffffu, pre, d);
      K += __shfl_down_sync(0xffffffffu, K, d);
      bad += __shfl_down_sync(0xffffffffu, bad, d);
    }
    if (threadIdx.x == 0) {
      s_tot[0] = pre;
      s_tot[1] = K;
      s_tot[2] = bad;
      s_tot[3] = window ? tail - head : wL;
      s_tot[4] = window ? head : wH;
    }
  }
  __syncthreads();
  const unsigned long long K = s_tot[1];
  const unsigned long long L = s_tot[3], qhead = s_tot[4];
  const unsigned long long Tq = L + K;
  const unsigned long long npop = a.flush ? Tq : (Tq / a.batch_size) * a.batch_size;
  if (npop > a.cap) {
    // refused: the claims are released; the window keeps its compaction
    if (!window) {
#pragma unroll
      for (int k = 0; k < RB_ITEMS; ++k)
        if (a.cand && ((flags >> k) & 1u)) a.slot[g.c[k]].phase = WAIT_UNCLAIMED;
    } else if (threadIdx.x == 0) {
      plan_reservation(a, head, tail, tail0, K, s_tot[2]);   // records the refusal
    }
    return;
  }
  // entries queued by earlier calls leave first: the Call's T + 1 CTAs take
  // a slice each (positions below L, apart from the new entries' L and up)
  {
    const unsigned long long n_old = L < npop ? L : npop;
    const unsigned long long per = (n_old + T) / (T + 1), j0 = (unsigned long long)b * per;
    const unsigned long long j1 = j0 + per < n_old ? j0 + per : n_old;
    for (unsigned long long j = j0 + threadIdx.x; j < j1; j += RB_THREADS) {
      const uint32_t c = a.queue[qhead + j];
      a.batched[j] = c;
      a.slot[c].phase = (a.slot[c].phase & ~3u) | PH_INFLIGHT;
    }
  }
  if (!window) {
    uint32_t rowpfx[RB_ITEMS];
    rank_rows(flags, s_rows, rowpfx);
#pragma unroll
    for (int k = 0; k < RB_ITEMS; ++k) {
      if (!((flags >> k) & 1u)) continue;
      const uint32_t c = g.c[k];
      const unsigned long long j = L + s_tot[0] + rowpfx[k];   // position in the logical queue
      if (j < npop) {
        a.batched[j] = c;
        a.slot[c].phase = ph_make(PH_INFLIGHT, 0u);
      } else {
        a.queue[qhead + j] = c;
        a.slot[c].phase = ph_make(PH_READY, 0u);
      }
    }
  } else if (threadIdx.x == 0) {
    plan_reservation(a, head, tail, tail0, K, s_tot[2]);
  }
}

__global__ void __launch_bounds__(RB_THREADS) ready_fused_kernel(ReadyArgs a) {
  fused_admit(a, gridDim.x - 1u, blockIdx.x, a.rs);
}

// Several Calls' admissions from one candidate list: the grid holds each
// Call's T tiles and its window CTA in turn.
__global__ void __launch_bounds__(RB_THREADS) ready_fused_calls_kernel(MultiReadyArgs m) {
  const uint32_t per = gridDim.x / m.n;   // CTAs per Call
  const uint32_t k = blockIdx.x / per, b = blockIdx.x % per;
  fused_admit(m.a[k], per - 1u, b, m.a[0].rs);
}

void launch_ready(const LaunchCfg& L, const ReadyArgs& a) {
  const uint64_t per = (uint64_t)RB_THREADS * RB_ITEMS;
  const uint64_t n_tiles = ceil_div(a.n_cand, per);
  if (!a.parent_bound && n_tiles + 1 <= (uint64_t)L.grid_rb_coop) {
    launch_coop(L, K_RB_FUSED, ready_fused_kernel, (int)n_tiles + 1, RB_THREADS, a);
    return;
  }
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

void launch_ready_calls(const LaunchCfg& L, const MultiReadyArgs& m) {
  const uint64_t per = ceil_div(m.a[0].n_cand, (uint64_t)RB_THREADS * RB_ITEMS) + 1;
  launch_coop(L, K_RB_FUSED, ready_fused_calls_kernel, (int)(per * m.n), RB_THREADS, m);
}

const void* kernel_ptr_ready(int which) {
  if (which == K_RB_FUSED_CALLS) return (const void*)ready_fused_calls_kernel;
  if (which == K_RB_FUSED) return (const void*)ready_fused_kernel;
  return which == K_RB_COUNT ? (const void*)ready_count_kernel : (const void*)ready_scatter_kernel;
}

}  // namespace ro
