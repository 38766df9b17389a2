// ro_common.cuh — layouts and device helpers shared by the lineage kernels.
//
// Per-child state of an expansion lives in two arrays:
//   slot[c]   16 bytes, one 32-byte sector holds it whole:
//             phase  uint32 Grain phase word (Eq. 2): bits 0-1 phase; for
//                    WAITING the upper 30 bits hold the admission claim of
//                    the current ro_batch_ready call (all ones = unclaimed),
//                    otherwise the attempt generation (Eq. 3);
//             len    payload length of the published result;
//             w      the arena offset (48 bits), the published outcome
//                    (3 bits), commit bookkeeping flags and the Call (8 bits).
//             The fence CAS, the Call check and the publish of a result
//             touch this one sector.
//   par[c]    uint32 immediate parent, written once at expansion.
// Per-parent state: pw[p] = remaining unsealed members (low 32 bits) plus the
// number of Failed/Suppressed members (high 32 bits), so one 64-bit atomic add
// both counts a member down and records its outcome class.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace ro {

// Completion streams a context plans its commits on (consecutive commits
// take them in turn), at most FIN_MAX; tile-status slots of the scans.
#ifndef RO_FIN_STREAMS
#define RO_FIN_STREAMS 3
#endif
constexpr int FIN_MAX = 4;
constexpr int FIN_STREAMS = RO_FIN_STREAMS;
static_assert(FIN_STREAMS >= 1 && FIN_STREAMS <= FIN_MAX, "1 to 4 completion streams");
constexpr int N_TILE_SLOTS = 10;

// ---- Grain phases (Eq. 2) -------------------------------------------------
constexpr uint32_t PH_WAITING = 0u, PH_READY = 1u, PH_INFLIGHT = 2u, PH_SEALED = 3u;
constexpr uint32_t CLAIM_NONE = 0x3FFFFFFFu;              // unclaimed WAITING
constexpr uint32_t WAIT_UNCLAIMED = (CLAIM_NONE << 2) | PH_WAITING;
constexpr uint64_t MAX_CAND = (uint64_t)CLAIM_NONE - 1;   // candidates per call

__host__ __device__ constexpr uint32_t ph_make(uint32_t phase, uint32_t gen) {
  return (gen << 2) | phase;
}

// ---- Item outcomes (Eq. 1) and report verdicts (Eq. 3) --------------------
constexpr uint8_t ST_PENDING = 0, ST_PRESENT = 1, ST_DROPPED = 2, ST_FAILED = 3,
                  ST_SUPPRESSED = 4;
// report kind (Section 4.4): the Grain failed and its open siblings are suppressed
constexpr uint8_t ST_GROUP_FAILURE = 5;
constexpr uint8_t V_ACCEPT = 0, V_INVALID = 1, V_NOT_INFLIGHT = 2, V_STALE = 3,
                  V_DUPLICATE = 4, V_BARRIER = 5;
// internal verdict: the Grain was SEALED at the same generation; resolved to
// ACCEPT or DUPLICATE by the commit's ordering pass
constexpr uint8_t V_DUP_CANDIDATE = 6;

// ---- per-child slot -----------------------------------------------------------
struct __align__(16) Slot {
  uint32_t phase;
  uint32_t len;
  uint64_t w;   // off (0-47) | state (48-50) | barrier (53) | sealer-seen (54) | conflict (55) |
                // call (56-63)
};
constexpr uint64_t W_OFF_MASK = (1ull << 48) - 1;
constexpr int W_STATE_SHIFT = 48;
constexpr uint64_t W_STATE_MASK = 7ull << W_STATE_SHIFT;
constexpr uint64_t W_BARRIER_BIT = 1ull << 53;   // sealed by a sibling's GroupFailure
constexpr uint64_t W_SEALER_BIT = 1ull << 54;
constexpr uint64_t W_CONFLICT_BIT = 1ull << 55;
constexpr int W_CALL_SHIFT = 56;
constexpr uint64_t MAX_ARENA = 1ull << 48;
// A parent with at least this many children is heavy.  When heavy parents
// hold a quarter of an expansion's children or more, a commit counts their
// members down in shared memory per CTA and adds them to the parent's
// counter once per CTA (their reports seldom share a warp), and takes their
// parent from the fill-tile table instead of the per-child parent array.
constexpr uint32_t HEAVY_CHILDREN = 4096;

__device__ __forceinline__ uint8_t w_state(uint64_t w) {
  return (uint8_t)((w >> W_STATE_SHIFT) & 7u);
}
__device__ __forceinline__ uint64_t w_off(uint64_t w) { return w & W_OFF_MASK; }
__device__ __forceinline__ uint32_t w_call(uint64_t w) { return (uint32_t)(w >> W_CALL_SHIFT); }

// ---- per-parent word ----------------------------------------------------------
__device__ __forceinline__ uint32_t pw_remaining(uint64_t v) { return (uint32_t)v; }
__device__ __forceinline__ uint32_t pw_bad(uint64_t v) { return (uint32_t)(v >> 32); }

// ---- errors recorded by kernels (sticky in DevScalars::err) --------------------
enum : uint32_t {
  ERR_CAPACITY = 1u,
  ERR_TIMEOUT = 2u,
  ERR_OVERFLOW = 4u,
  ERR_INVAL = 8u,
  // a copy CTA that gave up waiting exited with bulk copies into its shared
  // memory possibly still in flight (only after ERR_TIMEOUT)
  ERR_DRAIN = 16u,
};

// Header of a list of completed parents to assemble (see ListBufs).
struct ListHdr {
  unsigned long long n;      // listed parents
  unsigned long long M;      // members of the listed Present parents
  uint32_t err;              // the list cannot be planned (capacity)
  uint32_t pad;
  unsigned long long incomplete;   // listed entries that are not complete parents
};
// Header of an assembly plan (see PlanBufs).
struct PlanHdr {
  unsigned long long n;      // listed parents
  unsigned long long bytes;  // bytes to assemble
  unsigned long long nnz;    // members that contribute bytes
  uint32_t err;              // the plan is void (a capacity or arena check failed)
  uint32_t chunks_ok;        // the chunk table covers every chunk
  unsigned long long M;      // list entries (members of the listed Present parents)
  unsigned long long incomplete;   // listed entries that are not complete parents
  unsigned long long max_end;      // largest arena end of a planned member, when the
                                   // plan did not check it against the arena (else 0)
};

// Counters and small results that kernels hand to later kernels and to the
// host.  One instance per context, in device memory, mirrored to pinned host
// memory when a call synchronises.
struct DevScalars {
  uint32_t err;
  uint32_t pad0;
  unsigned long long stats[13];  // same order as ro_stats
  // ro_expand
  unsigned long long n_children, n_empty, last_nonempty_parent,
      n_heavy;   // children of parents with at least HEAVY_CHILDREN children
  // ro_gather_commit
  unsigned long long cm_n, cm_n_done[FIN_MAX];   // completed parents, per plan slot
  // per commit, in two slots (commit sequence & 1): duplicate candidates and
  // accepted GroupFailures the scatter saw; the next commit's scatter clears
  // the slot after this one
  unsigned long long cm_conflicts[2], cm_gf[2];
  // ro_retry
  unsigned long long rt_done;
  // ro_batch_ready_parent: the queue window after admission, the first short
  // chunk (no flush), totals, the admission's bad candidates, refusal
  unsigned long long pb_Q, pb_head, pb_old_tail, pb_stop, pb_npop, pb_nb, pb_R, pb_bad;
  uint32_t pb_err, pb_pad;
  uint32_t cm_pad0, cm_pad1;
  // ro_assemble
  unsigned long long as_bytes;    // bytes of the latest assemble (host read-back)
  unsigned long long as_elems;    // list entries of the latest assemble (host read-back)
  // dynamic tile counters / exit tickets / scan epochs, one per look-back kernel
  uint32_t tile_ctr[N_TILE_SLOTS];
  uint32_t exit_ctr[N_TILE_SLOTS];
  unsigned long long epoch[N_TILE_SLOTS];
};
// Admission scalars of one Call (ro_batch_ready): the first pass's counts,
// its exit ticket and the reservation it plans, the scatter pass's tile
// counter, exit ticket and scan epoch, and the one-pass admission's grid
// barrier.  One per Call, so that admissions of
// different Calls can run at the same time on streams of their own.
struct alignas(128) ReadyScalars {
  unsigned long long rb_kept, rb_bad, rb_L, rb_k, rb_npop, rb_head, rb_tail, rb_n_batches;
  unsigned long long epoch;
  uint32_t rb_ticket, rb_err, tile_ctr, exit_ctr;
  // one-pass admission: grid barrier (arrivals, generation)
  uint32_t bar_count, bar_gen;
};
// TS_COMMIT, TS_COMMIT_ODD, TS_COMMIT_2, TS_COMMIT_3: the completion lists
// and plans of commits whose sequence number is 0, 1, 2, 3 modulo the
// completion streams (they may run at the same time, one per stream);
// 5: asm_copy's exit ticket.
enum TileSlot { TS_EXPAND = 0, TS_COMMIT_ODD = 1, TS_COMMIT = 2, TS_ASM_PARENTS = 3,
                TS_ASM_MEMBERS = 4, TS_RETRY = 6, TS_PARENT = 7, TS_COMMIT_2 = 8, TS_COMMIT_3 = 9 };
__host__ __device__ constexpr int commit_slot(int pslot) {
  return pslot == 0 ? TS_COMMIT : pslot == 1 ? TS_COMMIT_ODD : pslot == 2 ? TS_COMMIT_2 : TS_COMMIT_3;
}

// Wait until the grid this launch depends on (programmatic dependent launch)
// has completed and its memory is visible; a no-op without a dependency.
__device__ __forceinline__ void wait_predecessor() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}
// Let the next kernel on the stream be scheduled now: it starts, and then
// waits in wait_predecessor() until this grid has finished and its memory is
// visible, so its launch overlaps this grid instead of following it.
__device__ __forceinline__ void allow_successor() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// ---- memory-order helpers --------------------------------------------------------
__device__ __forceinline__ uint32_t ld_acquire(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void st_release(uint32_t* p, uint32_t v) {
  asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ unsigned long long ld_relaxed_u64(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}

// ---- values carried by decoupled look-back scans ------------------------------------
struct Pair64 {
  unsigned long long a, b;
  __device__ __forceinline__ Pair64 operator+(const Pair64& o) const { return {a + o.a, b + o.b}; }
};

// Four 64-bit values carried together; the fourth combines by maximum.
struct Quad64 {
  unsigned long long a, b, c, d;
  __device__ __forceinline__ Quad64 operator+(const Quad64& o) const {
    return {a + o.a, b + o.b, c + o.c, d > o.d ? d : o.d};
  }
};

__device__ __forceinline__ unsigned long long load_cg(const unsigned long long* p) {
  return __ldcg(p);
}
__device__ __forceinline__ Pair64 load_cg(const Pair64* p) {
  return Pair64{__ldcg(&p->a), __ldcg(&p->b)};
}
__device__ __forceinline__ Quad64 load_cg(const Quad64* p) {
  return Quad64{__ldcg(&p->a), __ldcg(&p->b), __ldcg(&p->c), __ldcg(&p->d)};
}

// Spin limit of every device-side wait: ~2^22 polls with a short sleep each
// (well under a second).  A wait that runs out records ERR_TIMEOUT and the
// kernel carries on with what it has, so the context stays usable.
constexpr uint32_t SPIN_LIMIT = 1u << 22;

// Tile status for a single-pass scan: flag[t] = (epoch << 2) | kind with
// kind 1 = aggregate of tile t published, 2 = inclusive prefix published.
// The epoch is read from device memory at kernel start and advanced by the
// kernel's last CTA, so flags of earlier launches (or of earlier replays of
// a captured CUDA graph) never look current; nothing needs clearing.
template <class T>
struct TileStatus {
  unsigned long long* flag;
  T* agg;
  T* inc;
};

__device__ __forceinline__ unsigned long long ld_acquire_u64(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void st_release_u64(unsigned long long* p, unsigned long long v) {
  asm volatile("st.release.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}

template <class T>
__device__ __forceinline__ void ts_publish(const TileStatus<T>& ts, uint32_t tile, const T& v,
                                           unsigned long long kind, unsigned long long epoch) {
  if (kind == 1ull)
    ts.agg[tile] = v;
  else
    ts.inc[tile] = v;
  st_release_u64(ts.flag + tile, (epoch << 2) | kind);   // orders the value before the flag
}

__device__ __forceinline__ unsigned long long warp_sum(unsigned long long v) {
#pragma unroll
  for (int d = 16; d > 0; d >>= 1) v += __shfl_xor_sync(0xffffffffu, v, d);
  return v;
}
__device__ __forceinline__ Quad64 warp_sum(Quad64 v) {
#pragma unroll
  for (int d = 16; d > 0; d >>= 1) {
    Quad64 o;
    o.a = __shfl_xor_sync(0xffffffffu, v.a, d);
    o.b = __shfl_xor_sync(0xffffffffu, v.b, d);
    o.c = __shfl_xor_sync(0xffffffffu, v.c, d);
    o.d = __shfl_xor_sync(0xffffffffu, v.d, d);
    v = v + o;
  }
  return v;
}
__device__ __forceinline__ Pair64 warp_sum(Pair64 v) {
#pragma unroll
  for (int d = 16; d > 0; d >>= 1) {
    v.a += __shfl_xor_sync(0xffffffffu, v.a, d);
    v.b += __shfl_xor_sync(0xffffffffu, v.b, d);
  }
  return v;
}

// Exclusive prefix of tile `tile` given its local aggregate (decoupled
// look-back), computed by one whole warp: each step inspects the
// 32 * LB_PER_LANE nearest predecessors not yet summed at once (lane l the
// LB_PER_LANE after lane l - 1's), waits until every one up to the nearest
// inclusive prefix is published, adds the aggregates up to that prefix and
// stops there, else moves 32 * LB_PER_LANE tiles back.  Tiles are claimed in increasing order by running CTAs, so
// every predecessor is resident or done and each wait ends; the waits are
// bounded anyway (SPIN_LIMIT) and record ERR_TIMEOUT.  Every lane returns
// the prefix.
#ifndef RO_LB_PER_LANE
#define RO_LB_PER_LANE 1
#endif
constexpr int LB_PER_LANE = RO_LB_PER_LANE;   // predecessors each lane inspects per step (4 measured slower: its polls cost more than the shorter walks save)
template <class T>
__device__ T lookback_exclusive(const TileStatus<T>& ts, uint32_t tile, const T& local,
                                unsigned long long epoch, uint32_t* err) {
  const int lane = threadIdx.x & 31;
  if (tile == 0) {
    if (lane == 0) ts_publish(ts, 0, local, 2ull, epoch);
    __syncwarp();
    return T{};
  }
  if (lane == 0) ts_publish(ts, tile, local, 1ull, epoch);
  T excl{};
  int64_t j = (int64_t)tile - 1;   // nearest predecessor not summed yet
  for (;;) {
    // lane l inspects predecessors j - LB_PER_LANE * l - q, nearest first;
    // those past tile 0 count as an inclusive prefix of zero
    const int64_t m0 = j - (int64_t)lane * LB_PER_LANE;
    unsigned long long f[LB_PER_LANE];
    uint32_t spins = 0;
    bool gave_up = false;
    int stop = 32, qi = LB_PER_LANE;
    for (;;) {
      // per lane, nearest first: the first predecessor not published yet
      // (nr) and the first inclusive prefix (qi)
      int nr = LB_PER_LANE;
      qi = LB_PER_LANE;
#pragma unroll
      for (int q = LB_PER_LANE - 1; q >= 0; --q) {
        f[q] = 2ull;
        if (m0 - q >= 0) f[q] = ld_acquire_u64(ts.flag + (m0 - q));
        const bool ready = m0 - q < 0 || ((f[q] >> 2) == epoch && (f[q] & 3ull) != 0ull);
        if (!ready) nr = q;
        else if ((f[q] & 3ull) == 2ull) qi = q;
      }
      if (qi > nr) qi = LB_PER_LANE;   // an inclusive prefix behind an unpublished tile
      // go on once every predecessor up to the nearest inclusive prefix is in
      const unsigned bm = __ballot_sync(0xffffffffu, nr < LB_PER_LANE && qi == LB_PER_LANE);
      const unsigned sm = __ballot_sync(0xffffffffu, qi < LB_PER_LANE);
      stop = sm ? __ffs(sm) - 1 : 32;
      const int blocked = bm ? __ffs(bm) - 1 : 32;
      if (stop < blocked || blocked == 32) break;
      ++spins;
      bool give = spins > SPIN_LIMIT;
      // once any wait of this context has given up, stop waiting at once
      if ((spins & 1023u) == 0u && lane == 0 && (ld_acquire(err) & ERR_TIMEOUT)) give = true;
      if (__any_sync(0xffffffffu, give)) {
        gave_up = true;
        break;
      }
      __nanosleep(64);
    }
    if (gave_up) {
      if (lane == 0) atomicOr(err, ERR_TIMEOUT);
      break;
    }
    T v{};
    if (lane <= stop) {
      const int na = lane < stop ? LB_PER_LANE : qi;   // aggregates before it
#pragma unroll
      for (int q = 0; q < LB_PER_LANE; ++q) {
        if (m0 - q < 0) continue;
        if (q < na)
          v = v + load_cg(ts.agg + (m0 - q));
        else if (q == na && lane == stop)
          v = v + load_cg(ts.inc + (m0 - q));
      }
    }
    excl = excl + warp_sum(v);
    if (stop < 32) break;
    j -= 32 * LB_PER_LANE;
  }
  if (lane == 0) ts_publish(ts, tile, excl + local, 2ull, epoch);
  __syncwarp();
  return excl;
}

// All CTAs of the grid meet here.  Arrivals count up in the low 16 bits of
// the count (a CTA passing `flag` also adds 1 << 16); the last one resets the
// count and advances the generation to `target` (the launch's first
// generation plus the barrier's number, read before any CTA could arrive),
// with bit 31 set when any CTA passed `flag`.  The others wait for it
// (bounded: a wait that gives up records ERR_TIMEOUT and the call's results
// are void).  Returns whether any CTA passed `flag`, to every thread.
constexpr uint32_t BAR_FLAG = 1u << 31;
__device__ __forceinline__ bool grid_barrier(ReadyScalars* rs, uint32_t target, uint32_t* err,
                                             bool flag = false) {
  __shared__ uint32_t s_flag;
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    const uint32_t add = 1u + (flag ? (1u << 16) : 0u);
    const uint32_t old = atomicAdd(&rs->bar_count, add);
    if ((old & 0xFFFFu) == gridDim.x - 1u) {
      const bool any = ((old + add) >> 16) != 0u;
      rs->bar_count = 0u;
      st_release(&rs->bar_gen, target | (any ? BAR_FLAG : 0u));
      s_flag = any;
    } else {
      uint32_t spins = 0, g;
      while (((g = ld_acquire(&rs->bar_gen)) & ~BAR_FLAG) != target) {
        if (++spins > SPIN_LIMIT) {
          atomicOr(err, ERR_TIMEOUT);
          break;
        }
        __nanosleep(32);
      }
      s_flag = (g & BAR_FLAG) != 0u;
    }
    __threadfence();
  }
  __syncthreads();
  return s_flag;
}

// Claim the next tile of a dynamically scheduled (persistent) kernel.
__device__ __forceinline__ uint32_t claim_tile(uint32_t* ctr) { return atomicAdd(ctr, 1u); }

// CTAs that take part in a persistent kernel: never more than there are work
// units, so small launches cost few atomics.  The others return at once.
__device__ __forceinline__ uint32_t participants(uint64_t units) {
  return (uint32_t)(units < (uint64_t)gridDim.x ? units : (uint64_t)gridDim.x);
}

// Exit ticket: an add with acquire-release semantics at GPU scope, so
// everything the CTA did before it (its thread 0 after a CTA barrier) is
// visible to whoever draws the last ticket, and that CTA sees it all.
__device__ __forceinline__ uint32_t ticket(uint32_t* ctr) {
  uint32_t old;
  asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;" : "=r"(old) : "l"(ctr) : "memory");
  return old;
}

// Called by thread 0 of every participating CTA on exit; the last one out
// resets the tile counter and advances the epoch for the next launch (the
// end of the grid publishes them).
__device__ __forceinline__ void retire_cta(DevScalars* ds, int slot, uint32_t n_part) {
  if (ticket(&ds->exit_ctr[slot]) == n_part - 1) {
    ds->tile_ctr[slot] = 0u;
    ds->exit_ctr[slot] = 0u;
    ds->epoch[slot] += 1ull;
  }
}

// ---- block-wide scans ---------------------------------------------------------------
template <class T>
__device__ __forceinline__ T warp_incl_scan(T v) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    T u = __shfl_up_sync(0xffffffffu, v, d);
    if (lane >= d) v += u;
  }
  return v;
}

// Block exclusive scan of one value per thread.  `smem` holds >= 33 T.
// Returns the exclusive prefix; *total receives the block sum.
template <class T>
__device__ T block_excl_scan(T v, T* smem, T* total) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  T inc = warp_incl_scan(v);
  if (lane == 31) smem[wid] = inc;
  __syncthreads();
  if (wid == 0) {
    T s = (lane < nw) ? smem[lane] : T(0);
    s = warp_incl_scan(s);
    if (lane < nw) smem[lane] = s;   // inclusive warp totals
  }
  __syncthreads();
  T base = (wid > 0) ? smem[wid - 1] : T(0);
  *total = smem[nw - 1];
  __syncthreads();
  return base + inc - v;
}

__device__ __forceinline__ unsigned long long shfl_up_u64(unsigned long long v, int d) {
  return __shfl_up_sync(0xffffffffu, v, d);
}

// Block exclusive scan of a pair of 64-bit values.
__device__ __forceinline__ Pair64 block_excl_scan_pair(Pair64 v, Pair64* smem, Pair64* total) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  Pair64 inc = v;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    unsigned long long ua = shfl_up_u64(inc.a, d), ub = shfl_up_u64(inc.b, d);
    if (lane >= d) {
      inc.a += ua;
      inc.b += ub;
    }
  }
  if (lane == 31) smem[wid] = inc;
  __syncthreads();
  if (wid == 0) {
    Pair64 s = (lane < nw) ? smem[lane] : Pair64{0, 0};
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      unsigned long long ua = shfl_up_u64(s.a, d), ub = shfl_up_u64(s.b, d);
      if (lane >= d) {
        s.a += ua;
        s.b += ub;
      }
    }
    if (lane < nw) smem[lane] = s;
  }
  __syncthreads();
  Pair64 base = (wid > 0) ? smem[wid - 1] : Pair64{0, 0};
  *total = smem[nw - 1];
  __syncthreads();
  return Pair64{base.a + inc.a - v.a, base.b + inc.b - v.b};
}

__host__ __device__ constexpr uint64_t ceil_div(uint64_t a, uint64_t b) { return (a + b - 1) / b; }

}  // namespace ro
