// k_commit.cu — ro_gather_commit kernels (Section 4.4, Eq. 3; Section 4.2, Reduce).
//
// commit_scatter  one thread per report.  The fence of Eq. (3) is a single
//                 compare-and-swap of the child's phase word from
//                 IN-FLIGHT(gen) to SEALED(gen); the winner publishes the
//                 outcome into the child's 16-byte record (one sector) and
//                 counts the member down at its parent with one 64-bit atomic
//                 add on (remaining | bad << 32).  Lanes of a warp that hit
//                 the same parent are merged first (__match_any_sync), so a
//                 hot parent sees one atomic per warp.  Members of heavy
//                 parents (>= HEAVY_CHILDREN children, whose reports seldom
//                 share a warp) are first summed per CTA in a shared-memory
//                 table and added to the parent once per CTA.  The add that
//                 takes `remaining` to zero completes the parent and sets its
//                 bit in a completion bitmap (the counter's high half then
//                 tells whether a member Failed or was Suppressed).
// commit_fix      after the scatter, on the same stream: when the call
//                 carried two reports for one Grain or a GroupFailure (rare)
//                 it orders the repeats and applies the barriers, so the
//                 result equals applying the reports one by one in array
//                 order; otherwise it returns at once.
// The completed list and its copy plan come next, from commit_plan
// (k_complete.cu), which may run on another stream while later commits'
// scatters run (commits take completion bitmaps in turn).
#include <algorithm>

#include "ro_internal.h"

#ifndef RO_FIX_EARLY
#define RO_FIX_EARLY 0
#endif

namespace ro {

constexpr uint8_t V_WIN_SEALER = 7, V_WIN_CAND = 8, V_LOSE_SEALER = 9, V_LOSE_CAND = 10;
// The GroupFailure barrier table: per parent (seq << 32) | ~r, r the lowest
// accepted GroupFailure report of commit seq (atomicMax keeps the lowest r of
// the newest commit); an entry of an older commit means no barrier, so the
// table never needs clearing.
__device__ __forceinline__ unsigned long long gb_tag(uint32_t seq, uint32_t r) {
  return ((unsigned long long)seq << 32) | (unsigned long long)(uint32_t)~r;
}
__device__ __forceinline__ bool gb_get(const CommitArgs& a, uint32_t p, uint32_t* r) {
  const unsigned long long v = __ldcg(a.gb + p);
  if ((uint32_t)(v >> 32) != a.seq) return false;
  *r = ~(uint32_t)v;
  return true;
}
__device__ __forceinline__ uint32_t fix_slot(const CommitArgs& a) { return a.seq & 1u; }
__device__ __forceinline__ void stat_add(unsigned long long* s, unsigned long long d) {
  if (d) atomicAdd(s, d);   // d may be a negative delta in two's complement
}


// record word read past L1 (other threads update it with atomics at L2)
__device__ __forceinline__ uint64_t ld_w(const Slot* rc) {
  return __ldcg((const unsigned long long*)&rc->w);
}

__device__ __forceinline__ uint64_t commit_count(const CommitArgs& a) {
  if (!a.d_n) return a.n_host;
  const uint64_t n = *a.d_n;
  return n < a.n_host ? n : a.n_host;
}

__device__ void resolve_duplicates(const CommitArgs& a, uint64_t n);
__device__ void resolve_barriers(const CommitArgs& a, uint64_t n);
__device__ void seal_open(const CommitArgs& a, uint32_t pp, int lane, unsigned long long* n_wait,
                          unsigned long long* n_fly);

#ifndef RO_CM_GROUPS
#define RO_CM_GROUPS 1
#endif
constexpr int CM_GROUPS = RO_CM_GROUPS;   // groups of 32 reports a warp has in flight per step (2 and 4 measured slower)

// Warm L2 with the lines of this warp's first CM_GROUPS groups of 32 reports while the previous
// kernel drains (addresses inside the report arrays' host-given length; L2 is
// coherent, so nothing read later can be stale).
__device__ __forceinline__ void prefetch_l2(const void* p) {
  asm volatile("prefetch.global.L2 [%0];" ::"l"(p));
}
__device__ __forceinline__ void prefetch_reports(const CommitArgs& a) {
  const int lane = threadIdx.x & 31;
  if (lane >= 6 * CM_GROUPS) return;
  const uint64_t n_warps = ((uint64_t)gridDim.x * blockDim.x) >> 5;
  const uint64_t w = ((uint64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const uint64_t r0 = (w + (uint64_t)(lane / 6) * n_warps) * 32;   // this lane's group
  if (r0 >= a.n_host) return;
  switch (lane % 6) {
    case 0: prefetch_l2(a.child + r0); break;
    case 1: prefetch_l2(a.len + r0); break;
    case 2: prefetch_l2(a.off + r0); break;
    case 3: if (r0 + 16 < a.n_host) prefetch_l2(a.off + r0 + 16); break;
    case 4: prefetch_l2(a.state + r0); break;
    default: if (a.gen) prefetch_l2(a.gen + r0); break;
  }
}

// Per-CTA table of heavy parents' member counts (open addressing on the
// parent id): value = bad members << 32 | members, added to the parent's
// counter (as bad << 32 - members) when the CTA is done.
constexpr int HT_SIZE = 2048;
constexpr int HT_PROBES = 32;
constexpr uint32_t HT_EMPTY = 0xFFFFFFFFu;   // no parent has this id (P < 2^32)
struct HeavyTable {
  uint32_t key[HT_SIZE];
  unsigned long long val[HT_SIZE];
};
size_t commit_scatter_smem(int heavy) { return heavy ? sizeof(HeavyTable) : 0; }

// Count n_tot members (n_bad of them Failed or Suppressed) down at parent p;
// the add that takes `remaining` to zero completes the parent.
__device__ __forceinline__ void count_down(const CommitArgs& a, uint32_t p, uint32_t n_tot, uint32_t n_bad) {
  const unsigned long long delta = ((unsigned long long)n_bad << 32) - (unsigned long long)n_tot;
  const unsigned long long old = atomicAdd(a.pw + p, delta);
  if ((uint32_t)old == n_tot)   // the last members: the parent is complete
    atomicOr(a.bitmap + (p >> 5), 1u << (p & 31));
}

// Add to heavy parent p's entry of the CTA's table; false when no entry was
// found within HT_PROBES slots (the caller counts down directly).
__device__ __forceinline__ bool table_add(HeavyTable* t, uint32_t p, unsigned long long v) {
  uint32_t h = (p * 2654435761u) >> (32 - 11);   // HT_SIZE = 2^11
  for (int i = 0; i < HT_PROBES; ++i) {
    const uint32_t k = atomicCAS(&t->key[h], HT_EMPTY, p);
    if (k == HT_EMPTY || k == p) {
      atomicAdd(&t->val[h], v);
      return true;
    }
    h = (h + 1) & (HT_SIZE - 1);
  }
  return false;
}

// at most 56 registers: a CTA (256 threads) fits beside two copy CTAs
__global__ void __maxnreg__(56) commit_scatter_kernel(CommitArgs a) {
  prefetch_reports(a);
  wait_predecessor();
  allow_successor();
  extern __shared__ __align__(16) unsigned char cm_smem[];
  HeavyTable* ht = reinterpret_cast<HeavyTable*>(cm_smem);
  if (a.heavy)
    for (int i = threadIdx.x; i < HT_SIZE; i += blockDim.x) {
      ht->key[i] = HT_EMPTY;
      ht->val[i] = 0ull;
    }
  // verdict counts: accept, invalid, not in flight, stale, -, barrier,
  // duplicate candidates, accepted GroupFailures
  __shared__ unsigned long long s_cnt[8];
  DevScalars* ds = a.ds;
  if (threadIdx.x < 8) s_cnt[threadIdx.x] = 0;
  __syncthreads();
  const uint64_t n = commit_count(a);
  if (a.d_n && *a.d_n > a.n_host && blockIdx.x == 0 && threadIdx.x == 0)
    atomicOr(&ds->err, ERR_INVAL);
  if (blockIdx.x == 0 && threadIdx.x == 0) {   // the next commit's slot (its last reader is done)
    ds->cm_conflicts[fix_slot(a) ^ 1u] = 0ull;
    ds->cm_gf[fix_slot(a) ^ 1u] = 0ull;
  }
  const int lane = threadIdx.x & 31;
  const uint64_t warp_global = ((uint64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const uint64_t n_warps = ((uint64_t)gridDim.x * blockDim.x) >> 5;
  uint32_t cnt[8] = {0, 0, 0, 0, 0, 0, 0, 0};
  // Each warp takes CM_GROUPS groups of 32 reports per step (group q at
  // base + q * stride): their loads, parents and fence CASes are all in flight
  // before the first verdict is used.
  const uint64_t stride = n_warps * 32;
  for (uint64_t base = warp_global * 32; base < n; base += CM_GROUPS * stride) {
    uint64_t c[CM_GROUPS], o[CM_GROUPS];
    uint32_t l[CM_GROUPS], g[CM_GROUPS], par[CM_GROUPS], cur[CM_GROUPS];
    uint8_t st[CM_GROUPS], v[CM_GROUPS];
    bool heavy[CM_GROUPS], won[CM_GROUPS];
#pragma unroll
    for (int q = 0; q < CM_GROUPS; ++q) {
      const uint64_t r = base + q * stride + lane;
      v[q] = 255;   // inactive lane
      if (r < n) {
        c[q] = a.child[r];
        st[q] = a.state[r];
        l[q] = a.len[r];
        o[q] = a.off[r];
        g[q] = a.gen ? a.gen[r] : 0u;
      }
    }
#pragma unroll
    for (int q = 0; q < CM_GROUPS; ++q) {
      const uint64_t r = base + q * stride + lane;
      heavy[q] = won[q] = false;
      par[q] = cur[q] = 0u;
      if (r >= n) continue;
      const uint8_t s = st[q];
      const bool valid_state = s >= ST_PRESENT && s <= ST_GROUP_FAILURE;
      const bool in_bounds =
          s != ST_PRESENT || (o[q] <= a.arena_bytes && (uint64_t)l[q] <= a.arena_bytes - o[q]);
      if (c[q] >= a.N || !valid_state || !in_bounds) {
        v[q] = V_INVALID;
        continue;
      }
      v[q] = 254;   // decided below
      // the parent, immutable.  A fill tile of FILL_TILE children that
      // starts with the same parent as the next one is one heavy parent's
      // (it has more than HEAVY_CHILDREN children): the small fill-tile
      // table, resident in L2, names it, and the report touches no sector
      // but its slot's.  Otherwise it is read alongside the fence.
      const uint64_t t = c[q] / FILL_TILE;
      if (a.heavy && t + 1 < a.n_fill_tiles) {
        const uint32_t f0 = __ldg(a.tfp + t), f1 = __ldg(a.tfp + t + 1);
        heavy[q] = f0 == f1;
        par[q] = heavy[q] ? f0 : a.par[c[q]];
      } else {
        par[q] = a.par[c[q]];
      }
      // Eq. (3): accept iff IN-FLIGHT at the report's generation
      const uint32_t want = ph_make(PH_INFLIGHT, g[q]);
      if (g[q] >> 30) {
        cur[q] = a.slot[c[q]].phase;   // no Grain ever reaches such a generation
      } else {
        cur[q] = atomicCAS(&a.slot[c[q]].phase, want, ph_make(PH_SEALED, g[q]));
        won[q] = cur[q] == want;
      }
    }
#pragma unroll
    for (int q = 0; q < CM_GROUPS; ++q) {
      const uint64_t r = base + q * stride + lane;
      uint32_t p = 0;
      bool bad = false;
      if (v[q] == 254) {
        const uint8_t s = st[q];
        if (won[q]) {
          v[q] = V_ACCEPT;
          const bool present = s == ST_PRESENT;
          // a GroupFailure's own Grain failed
          const uint8_t outcome = (s == ST_GROUP_FAILURE) ? ST_FAILED : s;
          Slot* rc = a.slot + c[q];
          rc->len = present ? l[q] : 0u;
          atomicOr((unsigned long long*)&rc->w,
                   (unsigned long long)((present ? (o[q] & W_OFF_MASK) : 0ull) |
                                        ((uint64_t)outcome << W_STATE_SHIFT)));
          p = par[q];
          bad = (s == ST_FAILED || s == ST_SUPPRESSED || s == ST_GROUP_FAILURE);
          if (s == ST_GROUP_FAILURE) atomicMax(a.gb + p, gb_tag(a.seq, (uint32_t)r));   // barrier
        } else if ((cur[q] & 3u) == PH_WAITING || (cur[q] & 3u) == PH_READY) {
          v[q] = V_NOT_INFLIGHT;
        } else if ((cur[q] >> 2) != g[q]) {
          v[q] = V_STALE;
        } else if (ld_w(a.slot + c[q]) & W_BARRIER_BIT) {
          v[q] = V_BARRIER;   // suppressed by a sibling's GroupFailure in an earlier call
        } else {
          // SEALED at this generation: a duplicate, possibly of a report of
          // this same call with a higher index (ordered by commit_fix)
          v[q] = V_DUP_CANDIDATE;
          atomicOr((unsigned long long*)&a.slot[c[q]].w, (unsigned long long)W_CONFLICT_BIT);
        }
      }
      if (r < n) a.code[r] = v[q];
      // merge the accepted lanes of this warp by parent, one atomic per parent
      const unsigned acc = __ballot_sync(0xffffffffu, v[q] == V_ACCEPT);
      const unsigned badm = __ballot_sync(0xffffffffu, v[q] == V_ACCEPT && bad);
      if (v[q] == V_ACCEPT) {
        const unsigned grp = __match_any_sync(acc, p);
        if (lane == __ffs(grp) - 1) {
          const unsigned n_tot = __popc(grp), n_bad = __popc(grp & badm);
          if (!(heavy[q] && table_add(ht, p, ((unsigned long long)n_bad << 32) | n_tot)))
            count_down(a, p, n_tot, n_bad);
        }
      }
      if (v[q] <= V_DUP_CANDIDATE) cnt[v[q]] += 1;
      // any GroupFailure report (it may still win an ordering of duplicates)
      if (r < n && v[q] != V_INVALID && st[q] == ST_GROUP_FAILURE) cnt[7] += 1;
    }
  }
  // statistics: accepted, invalid, not in flight, stale, barrier (duplicates
  // are counted by the finish pass), candidates for ordering, GroupFailures
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    uint32_t x = cnt[k];
    for (int d = 16; d > 0; d >>= 1) x += __shfl_down_sync(0xffffffffu, x, d);
    if (lane == 0 && x) atomicAdd(&s_cnt[k], (unsigned long long)x);
  }
  __syncthreads();
  if (a.heavy)   // the CTA's heavy-parent counts, one add per parent
    for (int i = threadIdx.x; i < HT_SIZE; i += blockDim.x) {
      const uint32_t p = ht->key[i];
      if (p == HT_EMPTY) continue;
      const unsigned long long v = ht->val[i];
      count_down(a, p, (uint32_t)v, (uint32_t)(v >> 32));
    }
  if (threadIdx.x == 0) {
    for (int k = 0; k < 4; ++k)
      if (s_cnt[k]) atomicAdd(&ds->stats[k], s_cnt[k]);
    if (s_cnt[5]) atomicAdd(&ds->stats[7], s_cnt[5]);
    if (s_cnt[6]) atomicAdd(&ds->cm_conflicts[fix_slot(a)], s_cnt[6]);
    if (s_cnt[7]) atomicAdd(&ds->cm_gf[fix_slot(a)], s_cnt[7]);
  }
}

// The barriers of a call without repeated reports, spread over the grid:
// each CTA takes tiles of FX_TILE reports.  A report after its parent's
// barrier report (table gb) is rejected: an accepted one's Grain becomes
// Suppressed by the barrier, one that met a WAITING or READY Grain meets a
// sealed one (the fence compares generations); and the warp holding a
// barrier's own GroupFailure report seals that parent's open siblings.  The
// two touch disjoint Grains (sealed by this call vs still open), and the
// parent's counters are only added to, so no order between them is needed;
// the result equals the one-CTA pass in array order.
constexpr uint32_t FX_TILE = 2048;
__device__ void apply_barriers_grid(const CommitArgs& a, uint64_t n) {
  DevScalars* ds = a.ds;
  __shared__ unsigned long long s_d[7];   // as in resolve_barriers
  if (threadIdx.x < 7) s_d[threadIdx.x] = 0;
  __syncthreads();
  const int lane = threadIdx.x & 31;
  const uint64_t tiles = ceil_div(n, (uint64_t)FX_TILE);
  for (uint64_t t = blockIdx.x; t < tiles; t += gridDim.x) {
    for (uint64_t base = t * FX_TILE; base < (t + 1) * FX_TILE; base += blockDim.x) {
      const uint64_t r = base + threadIdx.x;
      uint32_t p = 0, b = 0;
      bool under = false, trig = false;
      uint8_t v = V_INVALID;
      uint64_t c = 0;
      if (r < n) {
        v = a.code[r];
        if (v == V_ACCEPT || v == V_NOT_INFLIGHT) {
          c = a.child[r];
          p = a.par[c];
          if (gb_get(a, p, &b)) {
            under = r > b;
            trig = r == b;   // the barrier's own (accepted) GroupFailure report
          }
        }
      }
      if (under) {
        if (v == V_ACCEPT) {
          Slot* rc = a.slot + c;
          const uint64_t keep = ld_w(rc) & ~(W_OFF_MASK | W_STATE_MASK);
          rc->len = 0u;
          rc->w = keep | ((uint64_t)ST_SUPPRESSED << W_STATE_SHIFT) | W_BARRIER_BIT;
          const uint8_t st = a.state[r];
          if (!(st == ST_FAILED || st == ST_SUPPRESSED || st == ST_GROUP_FAILURE))
            atomicAdd(a.pw + p, 1ull << 32);   // its outcome class is now bad
          a.code[r] = V_BARRIER;
          atomicAdd(&s_d[0], ~0ull);
          atomicAdd(&s_d[4], 1ull);
          atomicAdd(&s_d[6], 1ull);
        } else {
          const uint32_t ph = __ldcg(&a.slot[c].phase);
          const uint32_t gen_c = ((ph & 3u) == PH_WAITING) ? 0u : (ph >> 2);
          const uint32_t g = a.gen ? a.gen[r] : 0u;
          const bool same = g == gen_c;
          a.code[r] = same ? V_BARRIER : V_STALE;
          atomicAdd(&s_d[1], ~0ull);
          atomicAdd(&s_d[same ? 4 : 2], 1ull);
        }
      }
      unsigned m = __ballot_sync(0xffffffffu, trig);
      while (m) {
        const int src = __ffs(m) - 1;
        m &= m - 1;
        seal_open(a, __shfl_sync(0xffffffffu, p, src), lane, &s_d[5], &s_d[6]);
      }
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    stat_add(&ds->stats[0], s_d[0]);
    stat_add(&ds->stats[2], s_d[1]);
    stat_add(&ds->stats[3], s_d[2]);
    stat_add(&ds->stats[7], s_d[4]);
    stat_add(&ds->stats[8], s_d[5]);
    stat_add(&ds->stats[9], s_d[6]);
  }
}

// After the scatter, on the same stream: reports of one Grain that met in
// this call are ordered (one CTA, array order) and GroupFailure barriers
// applied (one CTA after an ordering, else the whole grid), so the next
// commit and the completion scan (which may run on another stream) see
// final outcomes.  Returns at once when the scatter saw neither.  Kept out
// of the scatter so that the scatter's registers and shared memory stay small.
__global__ void __launch_bounds__(CM_THREADS) commit_fix_kernel(CommitArgs a) {
#if RO_FIX_EARLY
  // the next commit's scatter launches now (it waits for this grid before it
  // touches lineage state, and warms L2 with its reports meanwhile)
  allow_successor();
  wait_predecessor();
#else
  wait_predecessor();
  allow_successor();
#endif
  DevScalars* ds = a.ds;
  const unsigned long long dups = ds->cm_conflicts[fix_slot(a)], gfs = ds->cm_gf[fix_slot(a)];
  if (dups == 0ull && gfs == 0ull) return;
  const uint64_t n = commit_count(a);
  if (dups) {
    if (blockIdx.x == 0) {
      resolve_duplicates(a, n);
      if (gfs) resolve_barriers(a, n);
    }
    return;
  }
  apply_barriers_grid(a, n);
}

// Make the lowest-index report of each Grain that was reported more than once
// in this call the accepted one.  Run by one CTA, only when the scatter saw
// such reports.
__device__ void resolve_duplicates(const CommitArgs& a, uint64_t n) {
  DevScalars* ds = a.ds;
  __shared__ unsigned long long s_dups;
  if (threadIdx.x == 0) s_dups = 0;
  __syncthreads();
  // A: this call's sealer of a conflicted Grain marks itself and opens the
  //    minimum-index election in the record's len field with its own index
  for (uint64_t r = threadIdx.x; r < n; r += blockDim.x) {
    if (a.code[r] != V_ACCEPT) continue;
    Slot* rc = a.slot + a.child[r];
    if (ld_w(rc) & W_CONFLICT_BIT) {
      rc->len = (uint32_t)r;
      atomicOr((unsigned long long*)&rc->w, (unsigned long long)W_SEALER_BIT);
    }
  }
  __syncthreads();
  // B: candidates of Grains sealed in this call vote; the others are plain
  //    duplicates of an earlier call's publication
  for (uint64_t r = threadIdx.x; r < n; r += blockDim.x) {
    if (a.code[r] != V_DUP_CANDIDATE) continue;
    Slot* rc = a.slot + a.child[r];
    if (ld_w(rc) & W_SEALER_BIT) {
      atomicMin(&rc->len, (uint32_t)r);
    } else {
      a.code[r] = V_DUPLICATE;
      atomicAnd((unsigned long long*)&rc->w, ~(unsigned long long)W_CONFLICT_BIT);
      atomicAdd(&s_dups, 1ull);
    }
  }
  __syncthreads();
  // C: every contender learns whether it won
  for (uint64_t r = threadIdx.x; r < n; r += blockDim.x) {
    const uint8_t v = a.code[r];
    if (v != V_ACCEPT && v != V_DUP_CANDIDATE) continue;
    const Slot* rc = a.slot + a.child[r];
    if (!(ld_w(rc) & W_SEALER_BIT)) continue;
    const bool win = __ldcg(&rc->len) == (uint32_t)r;
    a.code[r] = (v == V_ACCEPT) ? (win ? V_WIN_SEALER : V_LOSE_SEALER)
                                : (win ? V_WIN_CAND : V_LOSE_CAND);
  }
  __syncthreads();
  // D: the winner writes the record; outcome classes move with it
  for (uint64_t r = threadIdx.x; r < n; r += blockDim.x) {
    const uint8_t v = a.code[r];
    if (v < V_WIN_SEALER || v > V_LOSE_CAND) continue;
    const uint8_t s = a.state[r];
    const bool bad = (s == ST_FAILED || s == ST_SUPPRESSED || s == ST_GROUP_FAILURE);
    const uint64_t c = a.child[r];
    Slot* rc = a.slot + c;
    const uint32_t p = a.par[c];
    if (v == V_WIN_SEALER || v == V_WIN_CAND) {
      const bool present = s == ST_PRESENT;
      const uint8_t outcome = (s == ST_GROUP_FAILURE) ? ST_FAILED : s;
      const uint64_t keep = ld_w(rc) & ~(W_OFF_MASK | W_STATE_MASK | W_SEALER_BIT | W_CONFLICT_BIT);
      rc->len = present ? a.len[r] : 0u;
      rc->w = keep | (present ? (a.off[r] & W_OFF_MASK) : 0ull) | ((uint64_t)outcome << W_STATE_SHIFT);
      if (v == V_WIN_CAND && bad) atomicAdd(a.pw + p, 1ull << 32);
    } else {
      if (v == V_LOSE_SEALER && bad) atomicAdd(a.pw + p, ~((1ull << 32) - 1));   // -(1 << 32)
      atomicAdd(&s_dups, 1ull);
    }
  }
  __syncthreads();
  // E: the verdicts become final (a parent's outcome class moved with its
  //    counter in D; the completion list reads it from there)
  for (uint64_t r = threadIdx.x; r < n; r += blockDim.x) {
    const uint8_t v = a.code[r];
    if (v < V_WIN_SEALER || v > V_LOSE_CAND) continue;
    a.code[r] = (v == V_WIN_SEALER || v == V_WIN_CAND) ? V_ACCEPT : V_DUPLICATE;
  }
  __syncthreads();
  if (threadIdx.x == 0) atomicAdd(&ds->stats[4], s_dups);
  __syncthreads();
}


// A barrier seals every sibling of parent pp that is still open (a whole
// warp, lane = its lane): Suppressed, barrier bit set, counted down at the
// parent; the parent then completes (with a failed member it gathers
// nothing).  Siblings sealed while WAITING or READY and while IN-FLIGHT are
// added to *n_wait and *n_fly (shared counters of the CTA).
__device__ void seal_open(const CommitArgs& a, uint32_t pp, int lane, unsigned long long* n_wait,
                          unsigned long long* n_fly) {
  const uint64_t c0 = a.offsets[pp], c1 = a.offsets[pp + 1];
  uint32_t k_wait = 0, k_fly = 0;
  for (uint64_t d = c0 + lane; d < c1; d += 32) {
    Slot* rc = a.slot + d;
    const uint32_t ph = __ldcg(&rc->phase);
    const uint32_t f = ph & 3u;
    if (f == PH_SEALED) continue;
    const uint32_t gen_d = (f == PH_WAITING) ? 0u : (ph >> 2);
    Slot sl;   // the whole slot in one store
    sl.phase = ph_make(PH_SEALED, gen_d);
    sl.len = 0u;
    sl.w = (ld_w(rc) & ~(W_OFF_MASK | W_STATE_MASK)) | ((uint64_t)ST_SUPPRESSED << W_STATE_SHIFT) |
           W_BARRIER_BIT;
    *rc = sl;
    if (f == PH_INFLIGHT) ++k_fly; else ++k_wait;
  }
  for (int sh = 16; sh > 0; sh >>= 1) {
    k_wait += __shfl_down_sync(0xffffffffu, k_wait, sh);
    k_fly += __shfl_down_sync(0xffffffffu, k_fly, sh);
  }
  if (lane == 0) {
    const unsigned long long k = (unsigned long long)k_wait + k_fly;
    if (k) {
      const unsigned long long old = atomicAdd(a.pw + pp, (k << 32) - k);
      if ((uint32_t)old == k)   // the barrier completes the parent
        atomicOr(a.bitmap + (pp >> 5), 1u << (pp & 31));
    }
    atomicAdd(n_wait, (unsigned long long)k_wait);
    atomicAdd(n_fly, (unsigned long long)k_fly);
  }
  __syncwarp();
}

// GroupFailure barriers (Section 4.4) of this call, applied as if the
// reports were taken one by one in array order.  Run by one CTA, after the
// duplicate ordering and only when the call carries a GroupFailure report.
// For each parent, the lowest accepted GroupFailure report b installs the
// barrier: sibling reports before b stand; those after b see their Grain
// sealed by the barrier; every sibling still unsealed is sealed Suppressed.
// The GroupFailure reports and the barrier parents (few) are kept in shared
// memory; the barriers sorted by first child, so a report's barrier is a
// search there on its child id.  The two passes over all reports load 16
// reports' fields per thread before acting on any.  Past GF_CAP
// GroupFailure reports in one call, a report's parent and barrier are read
// from global memory instead (slower, same result).
constexpr int GF_CAP = 128;
constexpr int RB_GROUP = 16;
__device__ void resolve_barriers(const CommitArgs& a, uint64_t n) {
  DevScalars* ds = a.ds;
  // counter deltas: accepted, not in flight, stale, duplicate, barrier,
  // suppressed while waiting/ready, suppressed while in flight
  __shared__ unsigned long long s_d[7];   // two's complement
  __shared__ uint32_t s_gr[GF_CAP], s_gp[GF_CAP];   // GroupFailure reports and their parents
  __shared__ uint32_t s_nf, s_ng;
  __shared__ uint32_t s_p[GF_CAP], s_b[GF_CAP];     // barriers: parent, report
  __shared__ unsigned long long s_c0[GF_CAP], s_c1[GF_CAP];
  __shared__ uint32_t s_sp[GF_CAP], s_sb[GF_CAP];   // the same, sorted by first child
  __shared__ unsigned long long s_sc0[GF_CAP], s_sc1[GF_CAP];
  if (threadIdx.x < 7) s_d[threadIdx.x] = 0;
  if (threadIdx.x == 0) {
    s_nf = 0;
    s_ng = 0;
  }
  __syncthreads();
  auto parent_of = [&](uint64_t r, uint32_t* p) -> bool {
    const uint64_t c = a.child[r];
    if (c >= a.N) return false;
    *p = a.par[c];
    return true;
  };
  // 0: the call's GroupFailure reports (with a valid child)
  for (uint64_t base = (uint64_t)threadIdx.x * RB_GROUP; base < n; base += (uint64_t)blockDim.x * RB_GROUP) {
    uint8_t sv[RB_GROUP];
#pragma unroll
    for (int j = 0; j < RB_GROUP; ++j) sv[j] = (base + j < n) ? a.state[base + j] : 0;
#pragma unroll
    for (int j = 0; j < RB_GROUP; ++j) {
      uint32_t p;
      if (sv[j] != ST_GROUP_FAILURE || !parent_of(base + j, &p)) continue;
      const uint32_t k = atomicAdd(&s_nf, 1u);
      if (k < GF_CAP) {
        s_gr[k] = (uint32_t)(base + j);
        s_gp[k] = p;
      }
    }
  }
  __syncthreads();
  const uint32_t nf = s_nf;
  const bool fast = nf <= GF_CAP;
  // 1: barrier index per parent from the final verdicts (a GroupFailure can
  //    have lost to an earlier duplicate of its Grain)
  if (fast) {
    for (uint32_t i = threadIdx.x; i < nf; i += blockDim.x) a.gb[s_gp[i]] = 0ull;
    __syncthreads();
    for (uint32_t i = threadIdx.x; i < nf; i += blockDim.x)
      if (a.code[s_gr[i]] == V_ACCEPT) atomicMax(a.gb + s_gp[i], gb_tag(a.seq, s_gr[i]));
    __syncthreads();
    for (uint32_t i = threadIdx.x; i < nf; i += blockDim.x) {
      const uint32_t r = s_gr[i], p = s_gp[i];
      uint32_t br;
      if (a.code[r] != V_ACCEPT || !gb_get(a, p, &br) || br != r) continue;
      const uint32_t k = atomicAdd(&s_ng, 1u);
      s_p[k] = p;
      s_b[k] = r;
      s_c0[k] = a.offsets[p];
      s_c1[k] = a.offsets[p + 1];
    }
  } else {
    for (uint64_t r = threadIdx.x; r < n; r += blockDim.x) {
      uint32_t p;
      if (a.state[r] == ST_GROUP_FAILURE && parent_of(r, &p)) a.gb[p] = 0ull;
    }
    __syncthreads();
    for (uint64_t r = threadIdx.x; r < n; r += blockDim.x) {
      uint32_t p;
      if (a.state[r] == ST_GROUP_FAILURE && a.code[r] == V_ACCEPT && parent_of(r, &p))
        atomicMax(a.gb + p, gb_tag(a.seq, (uint32_t)r));
    }
  }
  __syncthreads();
  const uint32_t ng = s_ng;
  if (fast) {   // sort the barriers by first child (rank sort; ranges are disjoint)
    for (uint32_t i = threadIdx.x; i < ng; i += blockDim.x) {
      uint32_t rank = 0;
      for (uint32_t j = 0; j < ng; ++j) rank += s_c0[j] < s_c0[i];
      s_sp[rank] = s_p[i];
      s_sb[rank] = s_b[i];
      s_sc0[rank] = s_c0[i];
      s_sc1[rank] = s_c1[i];
    }
  }
  __syncthreads();
  if (fast && ng == 0) return;   // every GroupFailure was rejected
  // the barrier (parent, report) a child falls under, if any
  auto barrier_of = [&](uint64_t c, uint32_t* p, uint32_t* b) -> bool {
    if (c >= a.N) return false;
    if (fast) {
      if (c < s_sc0[0]) return false;
      uint32_t lo = 0, hi = ng;
      while (hi - lo > 1) {
        const uint32_t mid = (lo + hi) >> 1;
        if (s_sc0[mid] <= c) lo = mid; else hi = mid;
      }
      if (c >= s_sc1[lo]) return false;
      const uint32_t pp = s_sp[lo];
      *p = pp;
      *b = s_sb[lo];
      return true;
    }
    const uint32_t pp = a.par[c];
    uint32_t bb;
    if (!gb_get(a, pp, &bb)) return false;
    *p = pp;
    *b = bb;
    return true;
  };
  // 2: reports after a barrier whose Grain the barrier found open: those the
  //    scatter accepted were in flight; those it found WAITING or READY now
  //    meet a sealed Grain and the fence compares generations
  for (uint64_t base = (uint64_t)threadIdx.x * RB_GROUP; base < n; base += (uint64_t)blockDim.x * RB_GROUP) {
    uint8_t cv[RB_GROUP];
    uint32_t chv[RB_GROUP];
#pragma unroll
    for (int j = 0; j < RB_GROUP; ++j) cv[j] = (base + j < n) ? a.code[base + j] : V_INVALID;
#pragma unroll
    for (int j = 0; j < RB_GROUP; ++j)
      chv[j] = (cv[j] == V_ACCEPT || cv[j] == V_NOT_INFLIGHT) ? a.child[base + j] : 0u;
#pragma unroll 1
    for (int j = 0; j < RB_GROUP; ++j) {
      const uint8_t v = cv[j];
      if (v != V_ACCEPT && v != V_NOT_INFLIGHT) continue;
      const uint64_t r = base + j, c = chv[j];
      uint32_t p, b;
      if (!barrier_of(c, &p, &b) || r <= b) continue;
      if (v == V_ACCEPT) {
        Slot* rc = a.slot + c;
        const uint64_t keep = ld_w(rc) & ~(W_OFF_MASK | W_STATE_MASK);
        rc->len = 0u;
        rc->w = keep | ((uint64_t)ST_SUPPRESSED << W_STATE_SHIFT) | W_BARRIER_BIT;
        const uint8_t st = a.state[r];
        if (!(st == ST_FAILED || st == ST_SUPPRESSED || st == ST_GROUP_FAILURE))
          atomicAdd(a.pw + p, 1ull << 32);   // its outcome class is now bad
        a.code[r] = V_BARRIER;
        atomicAdd(&s_d[0], ~0ull);
        atomicAdd(&s_d[4], 1ull);
        atomicAdd(&s_d[6], 1ull);
      } else {
        const uint32_t ph = __ldcg(&a.slot[c].phase);
        const uint32_t gen_c = ((ph & 3u) == PH_WAITING) ? 0u : (ph >> 2);
        const uint32_t g = a.gen ? a.gen[r] : 0u;
        const bool same = g == gen_c;
        a.code[r] = same ? V_BARRIER : V_STALE;
        atomicAdd(&s_d[1], ~0ull);
        atomicAdd(&s_d[same ? 4 : 2], 1ull);
      }
    }
  }
  __syncthreads();
  // 3: duplicates after a barrier of a Grain whose accepted report (2) just
  //    turned into a barrier rejection (only if this call had duplicates)
  const bool had_dups = ds->cm_conflicts[fix_slot(a)] != 0;
  for (uint64_t base = (uint64_t)threadIdx.x * RB_GROUP; had_dups && base < n;
       base += (uint64_t)blockDim.x * RB_GROUP) {
    uint8_t cv[RB_GROUP];
#pragma unroll
    for (int j = 0; j < RB_GROUP; ++j) cv[j] = (base + j < n) ? a.code[base + j] : V_INVALID;
#pragma unroll 1
    for (int j = 0; j < RB_GROUP; ++j) {
      if (cv[j] != V_DUPLICATE) continue;
      const uint64_t r = base + j, c = a.child[r];
      uint32_t p, b;
      if (!barrier_of(c, &p, &b) || r <= b) continue;
      if (!(ld_w(a.slot + c) & W_BARRIER_BIT)) continue;   // sealed before the barrier
      a.code[r] = V_BARRIER;
      atomicAdd(&s_d[3], ~0ull);
      atomicAdd(&s_d[4], 1ull);
    }
  }
  __syncthreads();
  // 4: the barrier seals every sibling that is still open; one warp per
  //    barrier (the parent then completes; it has a failed member, so it
  //    gathers nothing)
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  if (fast) {
    for (uint32_t i = warp; i < ng; i += nw) seal_open(a, s_sp[i], lane, &s_d[5], &s_d[6]);
  } else {
    for (uint64_t base = (uint64_t)warp * 32; base < n; base += (uint64_t)nw * 32) {
      const uint64_t r = base + lane;
      uint32_t p = 0;
      uint32_t br = 0;
      const bool trig = r < n && a.state[r] == ST_GROUP_FAILURE && a.code[r] == V_ACCEPT &&
                        parent_of(r, &p) && gb_get(a, p, &br) && br == (uint32_t)r;
      unsigned m = __ballot_sync(0xffffffffu, trig);
      while (m) {
        const int src = __ffs(m) - 1;
        m &= m - 1;
        seal_open(a, __shfl_sync(0xffffffffu, p, src), lane, &s_d[5], &s_d[6]);
      }
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    stat_add(&ds->stats[0], s_d[0]);
    stat_add(&ds->stats[2], s_d[1]);
    stat_add(&ds->stats[3], s_d[2]);
    stat_add(&ds->stats[4], s_d[3]);
    stat_add(&ds->stats[7], s_d[4]);
    stat_add(&ds->stats[8], s_d[5]);
    stat_add(&ds->stats[9], s_d[6]);
  }
  __syncthreads();
}

void launch_commit_scatter(const LaunchCfg& L, const CommitArgs& a) {
  const uint64_t warps = ceil_div(a.n_host, 32);
  const int grid =
      (int)std::max<uint64_t>(1, std::min<uint64_t>(ceil_div(warps, CM_THREADS / 32),
                                                    (uint64_t)L.grid_commit));
  launch_k(L, K_COMMIT, commit_scatter_kernel, grid, CM_THREADS, commit_scatter_smem(a.heavy), a);
  // the fix returns at once unless the scatter flagged the call; a grid for
  // the barriers of calls without repeated reports
  const int grid_fix = (int)std::max<uint64_t>(
      1, std::min<uint64_t>(ceil_div(a.n_host, (uint64_t)FX_TILE), (uint64_t)L.grid_commit));
  launch_k(L, K_CFIX, commit_fix_kernel, grid_fix, CM_THREADS, 0, a);
}

const void* kernel_ptr_commit(int which) {
  return which == K_CFIX ? (const void*)commit_fix_kernel : (const void*)commit_scatter_kernel;
}

}  // namespace ro
