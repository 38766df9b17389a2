// k_complete.cu — the completion list and the assembly plan of a commit
// (Section 4.2: a parent's Reduce fires once every member outcome is
// resolved; its value is the Present members' payloads concatenated by
// ordinal, or Suppressed).
//
// commit_plan  runs after a commit's scatter (and its fix-up), one pass over
//              the commit's completion bitmap in tiles of CP_WORDS words
//              (32 parents per word).  Per tile it finds the parents this
//              commit completed, their members to gather (the parent's size
//              from the offsets, or 0 when its counter records a Failed or
//              Suppressed member) and those members' records, then takes ONE
//              decoupled look-back over the tuple (parents | members << 32,
//              payload bytes, contributing members, largest arena end).
//              With that prefix it writes, in ascending parent order:
//                * the completed list (parent, outcome, member base, first
//                  child, member-tile table): the commit's output and what an
//                  explicit assembly of it plans from;
//                * the copy plan (each parent's output offset, each
//                  contributing member's output position and arena offset,
//                  the 16 KB chunk -> member table), relative to the start of
//                  the call's output, so ro_assemble on the commit's list
//                  launches only the copy.
//              A small tile (at most CP_CAP completed parents and CP_ROUND
//              members) keeps its parents and its members' bytes and arena
//              offsets in shared memory across the look-back, so it reads
//              each record once; a larger one works through its parents in
//              groups of CP_CAP and its members in rounds of CP_ROUND, reading
//              the records once to total the tile and again (from L2) to
//              place them.
#include <algorithm>

#include "ro_internal.h"

namespace ro {

namespace {

__device__ __forceinline__ uint32_t last_le32(const uint32_t* v, uint32_t lo, uint32_t hi, uint64_t x) {
  while (hi - lo > 1) {
    const uint32_t mid = lo + ((hi - lo) >> 1);
    if ((uint64_t)v[mid] <= x) lo = mid; else hi = mid;
  }
  return lo;
}

// Block-wide sums of two values and the maximum of a third (thread 0 gets the result).
__device__ __forceinline__ void block_reduce3(unsigned long long& a, unsigned long long& b,
                                              unsigned long long& m, unsigned long long (*s)[CP_THREADS / 32]) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
#pragma unroll
  for (int d = 16; d > 0; d >>= 1) {
    a += __shfl_xor_sync(0xffffffffu, a, d);
    b += __shfl_xor_sync(0xffffffffu, b, d);
    const unsigned long long o = __shfl_xor_sync(0xffffffffu, m, d);
    m = o > m ? o : m;
  }
  if (lane == 0) {
    s[0][wid] = a;
    s[1][wid] = b;
    s[2][wid] = m;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int k = 1; k < CP_THREADS / 32; ++k) {
      a += s[0][k];
      b += s[1][k];
      m = s[2][k] > m ? s[2][k] : m;
    }
  }
  __syncthreads();
}

// A completed parent's members to gather (its size, or 0 when a member
// Failed or was Suppressed: the parent is then Suppressed) and first child.
__device__ __forceinline__ void parent_info(const CommitArgs& a, uint32_t p, uint32_t* m,
                                            uint32_t* first) {
  const unsigned long long v = __ldcg(a.pw + p);
  const uint64_t o0 = __ldg(a.offsets + p), o1 = __ldg(a.offsets + p + 1);
  *m = pw_bad(v) ? 0u : (uint32_t)(o1 - o0);
  *first = (uint32_t)o0;
}

// Members gathered by the completed parents of bitmap word w (loads issued
// four parents at a time, so they overlap).
__device__ __forceinline__ uint32_t word_members(const CommitArgs& a, uint64_t w, uint32_t bits) {
  uint32_t sum = 0;
  while (bits) {
    constexpr int G = 4;
    uint32_t p[G], m[G], cf[G];
    int cnt = 0;
#pragma unroll
    for (int u = 0; u < G; ++u) {
      if (bits) {
        p[u] = (uint32_t)(w * 32 + (uint32_t)(__ffs(bits) - 1));
        bits &= bits - 1;
        cnt = u + 1;
      }
    }
#pragma unroll
    for (int u = 0; u < G; ++u)
      if (u < cnt) parent_info(a, p[u], &m[u], &cf[u]);
#pragma unroll
    for (int u = 0; u < G; ++u)
      if (u < cnt) sum += m[u];
  }
  return sum;
}

struct CpShared {
  Pair64 scan[33];
  uint32_t wp[CP_WORDS + 1];    // per word: local list index of its first completed parent
  uint32_t wmb[CP_WORDS + 1];   // per word: local member base of its first completed parent
  uint32_t par[CP_CAP];         // staged group: parent id
  uint32_t pmb[CP_CAP + 1];     // staged group: local member base (+ the group's end)
  uint32_t coff[CP_CAP];        // staged group: first child
  unsigned long long red[3][CP_THREADS / 32];
  // one-round tiles: each member's contributed bytes and arena offset,
  // kept from the first pass for the second (a thread's own items only)
  uint32_t clen[CP_ROUND];
  unsigned long long csrc[CP_ROUND];
  Quad64 prefix;
  uint32_t tile;
};

// Stage the completed parents of local list positions [g0, g1) of this tile:
// each thread walks its bitmap word's completed parents (their member counts
// loaded in batches, so the loads overlap) and keeps those in the group.
__device__ void stage_group(const CommitArgs& a, CpShared& sh, uint64_t w, uint32_t bits, uint32_t g0,
                            uint32_t g1) {
  if (!bits) return;   // (threads past the tile's words have none)
  const uint32_t lo = sh.wp[threadIdx.x], hi = sh.wp[threadIdx.x + 1];
  if (hi <= g0 || lo >= g1) return;
  uint32_t b = bits, li = lo, mb = sh.wmb[threadIdx.x];
  constexpr int G = 4;
  while (b && li < g1) {
    uint32_t p[G], m[G], cf[G];
    int cnt = 0;
#pragma unroll
    for (int u = 0; u < G; ++u) {
      if (b) {
        p[u] = (uint32_t)(w * 32 + (uint32_t)(__ffs(b) - 1));
        b &= b - 1;
        cnt = u + 1;
      }
    }
#pragma unroll
    for (int u = 0; u < G; ++u)
      if (u < cnt) parent_info(a, p[u], &m[u], &cf[u]);
#pragma unroll
    for (int u = 0; u < G; ++u) {
      if (u >= cnt) break;
      if (li >= g0 && li < g1) {
        const uint32_t k = li - g0;
        sh.par[k] = p[u];
        sh.pmb[k] = mb;
        sh.coff[k] = cf[u];
        if (li + 1 == g1) sh.pmb[k + 1] = mb + m[u];   // the group's member end
      }
      mb += m[u];
      ++li;
    }
  }
}

// The records of this thread's CP_ITEMS consecutive members of a round
// (tile-local member indices gt .. gt+CP_ITEMS-1 below mhi), with the staged
// parent each belongs to and whether it is that parent's first member.
struct MemberMap {
  uint32_t par[CP_ITEMS];   // staged index
  uint32_t first;           // bit k: member k is its parent's first
  uint32_t valid;           // bit k: member k exists
};

__device__ __forceinline__ MemberMap map_members(const CpShared& sh, uint32_t cnt, uint64_t gt,
                                                 uint64_t mhi) {
  MemberMap mm;
  mm.first = 0;
  mm.valid = 0;
  uint32_t i = 0;
  if (gt < mhi) i = last_le32(sh.pmb, 0u, cnt, gt);
#pragma unroll
  for (int k = 0; k < CP_ITEMS; ++k) {
    const uint64_t g = gt + k;
    mm.par[k] = i;
    if (g < mhi) {
      while (g >= sh.pmb[i + 1]) ++i;   // member-less parents share their successor's base
      mm.par[k] = i;
      mm.valid |= 1u << k;
      if (g == sh.pmb[i]) mm.first |= 1u << k;
    }
  }
  return mm;
}

__device__ __forceinline__ void load_records(const CommitArgs& a, const CpShared& sh, const MemberMap& mm,
                                             uint64_t gt, Slot* rr) {
#pragma unroll
  for (int k = 0; k < CP_ITEMS; ++k) {
    if (mm.valid & (1u << k)) {
      const uint32_t i = mm.par[k];
      rr[k] = a.slot[(uint64_t)sh.coff[i] + (gt + k - sh.pmb[i])];
    } else {
      rr[k].len = 0;
      rr[k].w = 0;
    }
  }
}

__device__ __forceinline__ uint32_t contrib_of(const Slot& r) {
  return (w_state(r.w) == ST_PRESENT) ? r.len : 0u;
}

}  // namespace

__global__ void __maxnreg__(CP_MAXREG) commit_plan_kernel(CommitArgs a) {
  wait_predecessor();
  __shared__ CpShared sh;
  DevScalars* ds = a.ds;
  const ListBufs& L = a.list;
  const PlanBufs& pl = a.plan;
  const uint64_t n_words = ceil_div(a.P, 32);
  const uint64_t n_tiles = ceil_div(n_words, (uint64_t)CP_WORDS);
  if (n_tiles == 0) {
    if (blockIdx.x == 0 && threadIdx.x == 0) {
      ds->cm_n_done[a.pslot] = 0;
      L.hdr->n = 0;
      L.hdr->M = 0;
      L.hdr->err = 0u;
      L.hdr->incomplete = 0;
      L.mb[0] = 0;
      pl.off[0] = 0;
      pl.hdr->n = 0;
      pl.hdr->bytes = 0;
      pl.hdr->nnz = 0;
      pl.hdr->M = 0;
      pl.hdr->err = 0u;
      pl.hdr->chunks_ok = 1u;
      pl.hdr->incomplete = 0;
      pl.hdr->max_end = 0;
      if (a.n_done_out) *a.n_done_out = 0;
    }
    return;
  }
  const uint32_t n_part = participants(n_tiles);
  if (blockIdx.x >= n_part) return;
  const int slot = commit_slot(a.pslot);
  const unsigned long long epoch = ds->epoch[slot];

  for (;;) {
    if (threadIdx.x == 0) sh.tile = claim_tile(&ds->tile_ctr[slot]);
    __syncthreads();
    const uint32_t tile = sh.tile;
    __syncthreads();
    if (tile >= n_tiles) break;
    const uint64_t w = (uint64_t)tile * CP_WORDS + threadIdx.x;
    uint32_t bits = 0;
    if (threadIdx.x < CP_WORDS && w < n_words) bits = __ldcg(a.bitmap + w);
    const uint32_t wsum = word_members(a, w, bits);
    Pair64 tot;
    const Pair64 ex = block_excl_scan_pair(Pair64{(unsigned long long)__popc(bits), wsum}, sh.scan, &tot);
    if (threadIdx.x < CP_WORDS) {
      sh.wp[threadIdx.x] = (uint32_t)ex.a;
      sh.wmb[threadIdx.x] = (uint32_t)ex.b;
    }
    if (threadIdx.x == 0) {
      sh.wp[CP_WORDS] = (uint32_t)tot.a;
      sh.wmb[CP_WORDS] = (uint32_t)tot.b;
    }
    __syncthreads();
    const uint32_t Pt = (uint32_t)tot.a;
    const uint64_t Mt = tot.b;
    // one group and one round: parents stay staged, and the members' bytes
    // and offsets are kept in shared memory for the second pass
    const bool single = Pt <= CP_CAP && Mt <= CP_ROUND;

    // ---- pass 1: the tile's bytes, contributing members and largest arena end
    unsigned long long t_bytes = 0, t_nnz = 0, t_end = 0;
    for (uint32_t g0 = 0; g0 < Pt; g0 += CP_CAP) {
      const uint32_t g1 = min(Pt, g0 + CP_CAP), cnt = g1 - g0;
      stage_group(a, sh, w, bits, g0, g1);
      __syncthreads();
      const uint64_t mlo = sh.pmb[0], mhi = sh.pmb[cnt];
      for (uint64_t r0 = mlo; r0 < mhi; r0 += CP_ROUND) {
        const uint64_t gt = r0 + (uint64_t)threadIdx.x * CP_ITEMS;
        const MemberMap mm = map_members(sh, cnt, gt, mhi);
        Slot rr[CP_ITEMS];
        load_records(a, sh, mm, gt, rr);
#pragma unroll
        for (int k = 0; k < CP_ITEMS; ++k) {
          const uint32_t len = contrib_of(rr[k]);
          if (len) {
            t_bytes += len;
            t_nnz += 1;
            const unsigned long long e = w_off(rr[k].w) + len;
            t_end = e > t_end ? e : t_end;
          }
          if (single) {
            sh.clen[threadIdx.x * CP_ITEMS + k] = len;
            sh.csrc[threadIdx.x * CP_ITEMS + k] = w_off(rr[k].w);
          }
        }
      }
      if (!single) __syncthreads();   // the next group restages
    }
    block_reduce3(t_bytes, t_nnz, t_end, sh.red);
    if (threadIdx.x < 32) {   // one warp looks back
      Quad64 local{0, 0, 0, 0};
      if (threadIdx.x == 0) local = Quad64{(unsigned long long)Pt | (Mt << 32), t_bytes, t_nnz, t_end};
      local.a = __shfl_sync(0xffffffffu, local.a, 0);
      local.b = __shfl_sync(0xffffffffu, local.b, 0);
      local.c = __shfl_sync(0xffffffffu, local.c, 0);
      local.d = __shfl_sync(0xffffffffu, local.d, 0);
      const Quad64 pfx = lookback_exclusive(a.tsq, tile, local, epoch, &ds->err);
      if (threadIdx.x == 0) {
        sh.prefix = pfx;
        if (tile == n_tiles - 1) {   // the whole commit's totals
          const Quad64 all = pfx + local;
          const uint64_t n = all.a & 0xFFFFFFFFull, M = all.a >> 32;
          ds->cm_n_done[a.pslot] = n;
          L.hdr->n = n;
          L.hdr->M = M;
          L.hdr->err = 0u;
          L.hdr->incomplete = 0;
          L.mb[n] = (uint32_t)M;
          if (a.n_done_out) *a.n_done_out = n;
          pl.off[n] = all.b;
          pl.hdr->n = n;
          pl.hdr->bytes = all.b;
          pl.hdr->nnz = all.c;
          pl.hdr->M = M;
          pl.hdr->err = 0u;
          pl.hdr->incomplete = 0;
          pl.hdr->chunks_ok = ceil_div(all.b, AC_CHUNK) <= pl.ctfp_cap ? 1u : 0u;
          pl.hdr->max_end = all.d;
        }
      }
    }
    __syncthreads();
    const uint64_t gp = sh.prefix.a & 0xFFFFFFFFull, gm = sh.prefix.a >> 32;
    const uint64_t gb = sh.prefix.b, gz = sh.prefix.c;

    // ---- pass 2: the list entries and the plan
    uint64_t carry_b = 0, carry_z = 0;   // this tile's bytes / contributing members placed so far
    for (uint32_t g0 = 0; g0 < Pt; g0 += CP_CAP) {
      const uint32_t g1 = min(Pt, g0 + CP_CAP), cnt = g1 - g0;
      if (!single) {
        stage_group(a, sh, w, bits, g0, g1);
        __syncthreads();
      }
      // list entries of the group's parents
      for (uint32_t k = threadIdx.x; k < cnt; k += CP_THREADS) {
        const uint64_t i = gp + g0 + k;
        const uint32_t p = sh.par[k], m = sh.pmb[k + 1] - sh.pmb[k];
        const uint64_t mbg = gm + sh.pmb[k];
        a.done_int[i] = p;
        if (a.done_user) a.done_user[i] = p;
        L.status[i] = m ? ST_PRESENT : ST_SUPPRESSED;
        L.mb[i] = (uint32_t)mbg;
        L.coff[i] = sh.coff[k];
        for (uint64_t t = ceil_div(mbg, AM_TILE); t * AM_TILE < mbg + m && t < L.mtfp_cap; ++t)
          L.mtfp[t] = (uint32_t)i;
      }
      const uint64_t mlo = sh.pmb[0], mhi = sh.pmb[cnt];
      for (uint64_t r0 = mlo; r0 < mhi; r0 += CP_ROUND) {
        const uint64_t gt = r0 + (uint64_t)threadIdx.x * CP_ITEMS;
        const MemberMap mm = map_members(sh, cnt, gt, mhi);
        uint32_t clen[CP_ITEMS];
        uint64_t csrc[CP_ITEMS];
        if (single) {
#pragma unroll
          for (int k = 0; k < CP_ITEMS; ++k) {
            clen[k] = sh.clen[threadIdx.x * CP_ITEMS + k];
            csrc[k] = sh.csrc[threadIdx.x * CP_ITEMS + k];
          }
        } else {
          Slot rr[CP_ITEMS];
          load_records(a, sh, mm, gt, rr);
#pragma unroll
          for (int k = 0; k < CP_ITEMS; ++k) {
            clen[k] = contrib_of(rr[k]);
            csrc[k] = w_off(rr[k].w);
          }
        }
        Pair64 mine{0, 0};
#pragma unroll
        for (int k = 0; k < CP_ITEMS; ++k) {
          mine.a += clen[k];
          mine.b += clen[k] ? 1ull : 0ull;
        }
        Pair64 rtot;
        const Pair64 rex = block_excl_scan_pair(mine, sh.scan, &rtot);
        uint64_t pos = gb + carry_b + rex.a, j = gz + carry_z + rex.b;
#pragma unroll
        for (int k = 0; k < CP_ITEMS; ++k) {
          if (!(mm.valid & (1u << k))) break;
          const uint32_t i = mm.par[k];
          if (mm.first & (1u << k)) {
            // the parent starts here, and so do the member-less parents staged just before it
            const uint32_t g = sh.pmb[i];
            pl.off[gp + g0 + i] = pos;
            for (int32_t q = (int32_t)i - 1; q >= 0 && sh.pmb[q] == g; --q) pl.off[gp + g0 + q] = pos;
          }
          const uint32_t len = clen[k];
          if (len) {
            if (j < pl.member_cap) {
              pl.cpos[j] = pos;
              pl.csrc[j] = csrc[k];
            }
            for (uint64_t t = ceil_div(pos, AC_CHUNK); t * AC_CHUNK < pos + len && t < pl.ctfp_cap; ++t)
              pl.ctfp[t] = (uint32_t)j;
            pos += len;
            j += 1;
          }
        }
        carry_b += rtot.a;
        carry_z += rtot.b;
      }
      // member-less parents at the group's end start where its members end
      for (uint32_t k = threadIdx.x; k < cnt; k += CP_THREADS)
        if (sh.pmb[k] == mhi) pl.off[gp + g0 + k] = gb + carry_b;
      __syncthreads();   // the next group restages
    }
    if (bits) a.bitmap[w] = 0u;   // the bitmap slot is clean for its next commit
  }
  if (threadIdx.x == 0) retire_cta(ds, slot, n_part);
}

void launch_commit_plan(const LaunchCfg& L, const CommitArgs& a) {
  const uint64_t n_tiles = ceil_div(ceil_div(a.P, 32), (uint64_t)CP_WORDS);
  const int grid = (int)std::max<uint64_t>(1, std::min<uint64_t>(n_tiles, (uint64_t)L.grid_cplan));
  launch_k(L, K_CPLAN, commit_plan_kernel, grid, CP_THREADS, 0, a);
}

const void* kernel_ptr_complete() { return (const void*)commit_plan_kernel; }

}  // namespace ro
