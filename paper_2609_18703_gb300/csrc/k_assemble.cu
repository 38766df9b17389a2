// k_assemble.cu — ro_assemble kernels (Section 4.2, Reduce).
//
// A completed parent is Suppressed if a member Failed or was Suppressed,
// otherwise Present with the Present members' payloads concatenated by
// ordinal (Dropped members add nothing).  The work is a segmented byte gather
// from the result arena in three steps:
//   asm_parents  (caller's lists only; commit_plan does this for the
//                parents a commit completed) per listed parent: outcome,
//                members to gather (0 unless Present), their exclusive scan
//                (member bases), and for every AM_TILE-member tile the parent
//                holding its first member;
//   asm_members  per member, load-balanced over AM_TILE-member tiles so a
//                100k-member parent spreads over many CTAs: read the record,
//                scan the Present bytes (single-pass look-back) and write the
//                plan — each parent's relative output offset, each
//                contributing member's relative position and arena offset, and
//                for every 16 KB chunk of the output the member holding its
//                first byte;
//   asm_copy     per chunk: two producer warps stage chunks' member pieces
//                in shared memory with cp.async.bulk (a ring of AC_STAGES
//                stages, mbarrier completion, bounded waits) while eight
//                consumer warps turn staged chunks into aligned 16-byte
//                stores; source and destination alignments may differ
//                arbitrarily.
// The plan is independent of where the output starts, so planning (on the
// context's plan stream) can run ahead of the copies (copy stream).
#include <algorithm>

#include "ro_internal.h"

namespace ro {

constexpr int TS_ASM_COPY = 5;
#ifndef RO_COPY_DYNAMIC
#define RO_COPY_DYNAMIC 1
#endif

template <class V>
__device__ __forceinline__ uint32_t last_le_u(const V* v, uint32_t lo, uint32_t hi, uint64_t x) {
  while (hi - lo > 1) {
    const uint32_t mid = lo + ((hi - lo) >> 1);
    if ((uint64_t)v[mid] <= x)
      lo = mid;
    else
      hi = mid;
  }
  return lo;
}

// ---------------------------------------------------------------------------
// asm_parents: a caller's list -> outcomes, member bases, member-tile table.
__global__ void __launch_bounds__(AP_THREADS) asm_parents_kernel(AssembleArgs a) {
  wait_predecessor();
  __shared__ unsigned long long s_scan[33];
  __shared__ uint32_t s_tile;
  __shared__ unsigned long long s_prefix;
  __shared__ unsigned long long s_incomplete;
  DevScalars* ds = a.ds;
  const ListBufs& L = a.list;
  const uint64_t n_req = a.d_n ? *a.d_n : a.n_host;
  if (n_req > a.n_host) {   // a device count beyond the arrays' length
    if (blockIdx.x == 0 && threadIdx.x == 0) {
      L.hdr->err = 1u;
      L.hdr->n = 0;
      atomicOr(&ds->err, ERR_INVAL);
    }
    return;
  }
  const uint64_t n = n_req;
  const uint64_t TILE = (uint64_t)AP_THREADS * AP_ITEMS;
  const uint64_t n_tiles = ceil_div(n, TILE);
  if (n_tiles == 0) {
    if (blockIdx.x == 0 && threadIdx.x == 0) {
      L.mb[0] = 0;
      L.hdr->n = 0;
      L.hdr->M = 0;
      L.hdr->err = 0u;
    }
    return;
  }
  const uint32_t n_part = participants(n_tiles);
  if (blockIdx.x >= n_part) return;
  if (threadIdx.x == 0) s_incomplete = 0;
  for (;;) {
    if (threadIdx.x == 0) s_tile = claim_tile(&ds->tile_ctr[TS_ASM_PARENTS]);
    __syncthreads();
    const uint32_t tile = s_tile;
    __syncthreads();
    if (tile >= n_tiles) break;
    const uint64_t i0 = tile * TILE + (uint64_t)threadIdx.x * AP_ITEMS;
    uint32_t m[AP_ITEMS], cf[AP_ITEMS];
    unsigned long long mine = 0;
    uint32_t incomplete = 0;
#pragma unroll
    for (int k = 0; k < AP_ITEMS; ++k) {
      const uint64_t i = i0 + k;
      m[k] = 0;
      cf[k] = 0;
      if (i >= n) continue;
      const uint64_t p = L.parents[i];
      uint8_t st = ST_PENDING;
      if (p < a.P) {
        const unsigned long long v = a.pw[p];
        cf[k] = (uint32_t)a.offsets[p];
        if (pw_remaining(v) == 0u) {
          if (pw_bad(v) != 0u) {
            st = ST_SUPPRESSED;
          } else {
            st = ST_PRESENT;
            m[k] = (uint32_t)(a.offsets[p + 1] - a.offsets[p]);
          }
        }
      }
      if (st == ST_PENDING) ++incomplete;
      L.status[i] = st;
      mine += m[k];
    }
    if (incomplete) atomicAdd(&s_incomplete, (unsigned long long)incomplete);
    unsigned long long total;
    unsigned long long excl = block_excl_scan(mine, s_scan, &total);
    if (threadIdx.x < 32) {  // one warp looks back
      const auto pfx = lookback_exclusive(a.ts_parents, tile, total, ds->epoch[TS_ASM_PARENTS], &ds->err);
      if (threadIdx.x == 0) s_prefix = pfx;
    }
    __syncthreads();
    unsigned long long run = s_prefix + excl;
#pragma unroll
    for (int k = 0; k < AP_ITEMS; ++k) {
      const uint64_t i = i0 + k;
      if (i >= n) break;
      L.mb[i] = (uint32_t)run;
      L.coff[i] = cf[k];
      if (m[k]) {
        for (uint64_t b = ceil_div(run, AM_TILE); b * AM_TILE < run + m[k] && b < L.mtfp_cap; ++b)
          L.mtfp[b] = (uint32_t)i;
      }
      run += m[k];
    }
    if (tile == n_tiles - 1 && threadIdx.x == AP_THREADS - 1) {
      L.mb[n] = (uint32_t)run;
      L.hdr->n = n;
      L.hdr->M = run;
      // more members than the plan holds (a parent listed many times)
      L.hdr->err = run > a.plan.member_cap ? 1u : 0u;
      if (run > a.plan.member_cap) atomicOr(&ds->err, ERR_CAPACITY);
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    // counted once the assembly succeeds (asm_copy)
    if (s_incomplete) atomicAdd(&L.hdr->incomplete, s_incomplete);
    retire_cta(ds, TS_ASM_PARENTS, n_part);
  }
}

// ---------------------------------------------------------------------------
// asm_members: list -> plan (relative offsets and member positions).
__global__ void __maxnreg__(56) asm_members_kernel(AssembleArgs a) {
  wait_predecessor();
  __shared__ uint32_t s_mb[AM_SMEM_CAP];
  __shared__ uint32_t s_coff[AM_SMEM_CAP];
  __shared__ Pair64 s_scan[33];
  __shared__ uint32_t s_tile;
  __shared__ Pair64 s_prefix;
  DevScalars* ds = a.ds;
  const ListBufs& L = a.list;
  const PlanBufs& pl = a.plan;
  const ListHdr lh = *L.hdr;
  const uint64_t n = lh.n, M = lh.M;
  // the list's entries must fit the caller's list-structure outputs
  const bool elems_too_many = a.elem_base && M > a.elem_cap;
  if (lh.err || elems_too_many) {   // nothing to plan
    if (blockIdx.x == 0 && threadIdx.x == 0) {
      pl.hdr->n = n;
      pl.hdr->bytes = 0;
      pl.hdr->nnz = 0;
      pl.hdr->M = M;
      pl.hdr->incomplete = 0;
      pl.hdr->max_end = 0;
      pl.hdr->err = 1u;
      L.hdr->incomplete = 0;   // spent (asm_parents adds to it)
      if (elems_too_many) atomicOr(&ds->err, ERR_CAPACITY);
    }
    return;
  }
  const uint64_t n_tiles = ceil_div(M, AM_TILE);
  const uint64_t par_units = ceil_div(n, (uint64_t)AM_TILE);
  const uint32_t n_part = participants((n_tiles > par_units ? n_tiles : par_units) + 1);
  if (blockIdx.x >= n_part) return;
  if (a.elem_base) {   // each listed parent's first list entry (its member base)
    const uint64_t stride = (uint64_t)n_part * blockDim.x;
    for (uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; i <= n; i += stride)
      a.elem_base[i] = L.mb[i];
  }

  if (M == 0) {   // nothing to gather: every listed parent starts at 0
    const uint64_t stride = (uint64_t)n_part * blockDim.x;
    for (uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; i <= n; i += stride)
      pl.off[i] = 0;
    if (blockIdx.x == 0 && threadIdx.x == 0) {
      pl.hdr->n = n;
      pl.hdr->bytes = 0;
      pl.hdr->nnz = 0;
      pl.hdr->M = 0;
      pl.hdr->incomplete = lh.incomplete;
      pl.hdr->max_end = 0;
      pl.hdr->err = 0u;
      pl.hdr->chunks_ok = 1u;
      L.hdr->incomplete = 0;   // spent (asm_parents adds to it)
    }
    return;
  }

  for (;;) {
    if (threadIdx.x == 0) s_tile = claim_tile(&ds->tile_ctr[TS_ASM_MEMBERS]);
    __syncthreads();
    const uint32_t tile = s_tile;
    __syncthreads();
    if (tile >= n_tiles) break;
    const uint64_t g0 = (uint64_t)tile * AM_TILE;
    const uint64_t i_lo = L.mtfp[tile];
    const uint64_t i_hi = (tile + 1 < n_tiles) ? L.mtfp[tile + 1] : n - 1;
    const uint64_t R = i_hi - i_lo + 1;
    const bool staged = R <= AM_SMEM_CAP;
    if (staged) {
#pragma unroll 4
      for (uint32_t k = threadIdx.x; k < (uint32_t)R; k += AM_THREADS) {
        s_mb[k] = __ldcg(L.mb + i_lo + k);
        s_coff[k] = __ldcg(L.coff + i_lo + k);
      }
    }
    __syncthreads();

    // my members gt .. gt+AM_ITEMS-1 are consecutive: one search finds the
    // list entry holding the first, a walk over the member bases the rest
    const uint64_t gt = g0 + (uint64_t)threadIdx.x * AM_ITEMS;
    constexpr uint64_t NONE = ~0ull;
    uint64_t ridx[AM_ITEMS];
    uint32_t par[AM_ITEMS];
    uint32_t firsts = 0;   // bit k: member gt+k is its parent's first
    {
      uint64_t i = i_lo;
      if (gt < M) {
        if (staged) {
          i = i_lo + last_le_u(s_mb, 0u, (uint32_t)R, gt);
        } else {
          uint64_t lo = i_lo, hi = i_hi + 1;
          while (hi - lo > 1) {
            const uint64_t mid = lo + ((hi - lo) >> 1);
            if (L.mb[mid] <= gt) lo = mid; else hi = mid;
          }
          i = lo;
        }
      }
      // no member of this tile lies past entry i_hi
      auto mb_at = [&](uint64_t x) -> uint64_t { return staged ? s_mb[x - i_lo] : L.mb[x]; };
      uint64_t mbi = gt < M ? mb_at(i) : 0;
      uint64_t mbn = (gt < M && i < i_hi) ? mb_at(i + 1) : NONE;
      uint64_t cof = gt < M ? (staged ? s_coff[i - i_lo] : L.coff[i]) : 0;
#pragma unroll
      for (int k = 0; k < AM_ITEMS; ++k) {
        const uint64_t g = gt + k;
        ridx[k] = NONE;
        par[k] = (uint32_t)i;
        if (g < M) {
          while (g >= mbn) {   // member-less entries have equal bases and are passed over
            ++i;
            mbi = mbn;
            mbn = (i < i_hi) ? mb_at(i + 1) : NONE;
            cof = staged ? s_coff[i - i_lo] : L.coff[i];
          }
          par[k] = (uint32_t)i;
          if (g == mbi) firsts |= 1u << k;
          ridx[k] = cof + (g - mbi);
        }
      }
    }
    // all record loads first (no store in between), so they overlap
    Slot rr[AM_ITEMS];
#pragma unroll
    for (int k = 0; k < AM_ITEMS; ++k) {
      if (ridx[k] != NONE) {
        rr[k] = a.slot[ridx[k]];
      } else {
        rr[k].len = 0;
        rr[k].w = 0;
      }
    }
    uint32_t contrib[AM_ITEMS];
    uint64_t src[AM_ITEMS];
    Pair64 mine{0, 0};
#pragma unroll
    for (int k = 0; k < AM_ITEMS; ++k) {
      contrib[k] = 0;
      src[k] = 0;
      const Slot r = rr[k];
      if (w_state(r.w) == ST_PRESENT && r.len) {
        contrib[k] = r.len;
        src[k] = w_off(r.w);
        // the arena passed here must hold what the commit accepted
        if (src[k] > a.arena_bytes || (uint64_t)r.len > a.arena_bytes - src[k]) {
          atomicOr(&ds->err, ERR_INVAL);
          pl.hdr->err = 1u;
        }
      }
      mine.a += contrib[k];
      mine.b += contrib[k] ? 1ull : 0ull;
    }
    Pair64 total;
    Pair64 excl = block_excl_scan_pair(mine, s_scan, &total);
    if (threadIdx.x < 32) {  // one warp looks back
      const auto pfx = lookback_exclusive(a.ts_members, tile, total, ds->epoch[TS_ASM_MEMBERS], &ds->err);
      if (threadIdx.x == 0) s_prefix = pfx;
    }
    __syncthreads();
    Pair64 run = s_prefix + excl;   // (bytes, contributing members) before my first item
#pragma unroll
    for (int k = 0; k < AM_ITEMS; ++k) {
      const uint64_t g = gt + k;
      if (g >= M) break;
      const uint64_t pos = run.a;
      if (firsts & (1u << k)) {
        // the parent starts here, and so do the member-less parents listed just before it
        pl.off[par[k]] = pos;
        for (int64_t q = (int64_t)par[k] - 1; q >= 0; --q) {
          const uint32_t mbq = (staged && (uint64_t)q >= i_lo) ? s_mb[q - i_lo] : L.mb[q];
          if (mbq != g) break;
          pl.off[q] = pos;
        }
      }
      if (a.elem_base) {   // the member's list entry (offset relative until the copy)
        a.elem_state[g] = w_state(rr[k].w) == ST_PRESENT ? ST_PRESENT : ST_DROPPED;
        a.elem_len[g] = contrib[k];
        a.elem_off[g] = pos;
      }
      if (contrib[k]) {
        const uint64_t j = run.b;
        if (j < pl.member_cap) {
          pl.cpos[j] = pos;
          pl.csrc[j] = src[k];
        }
        const uint64_t e = pos + contrib[k];
        for (uint64_t t = ceil_div(pos, AC_CHUNK); t * AC_CHUNK < e && t < pl.ctfp_cap; ++t)
          pl.ctfp[t] = (uint32_t)j;
        run.b += 1;
        run.a += contrib[k];
      }
    }
    if (tile == n_tiles - 1 && threadIdx.x == AM_THREADS - 1) {
      pl.off[n] = run.a;
      for (int64_t q = (int64_t)n - 1; q >= 0; --q) {
        if ((uint64_t)L.mb[q] != M) break;   // member-less parents at the very end
        pl.off[q] = run.a;
      }
      pl.hdr->n = n;
      pl.hdr->bytes = run.a;
      pl.hdr->nnz = run.b;
      pl.hdr->M = M;
      pl.hdr->incomplete = lh.incomplete;
      pl.hdr->max_end = 0;   // checked here, member by member
      pl.hdr->chunks_ok = ceil_div(run.a, AC_CHUNK) <= pl.ctfp_cap ? 1u : 0u;
    }
    __syncthreads();
  }
  if (threadIdx.x == 0 && ticket(&ds->exit_ctr[TS_ASM_MEMBERS]) == n_part - 1) {
    ds->tile_ctr[TS_ASM_MEMBERS] = 0u;
    ds->exit_ctr[TS_ASM_MEMBERS] = 0u;
    ds->epoch[TS_ASM_MEMBERS] += 1ull;
    L.hdr->incomplete = 0;   // spent (asm_parents adds to it)
  }
}

// ---------------------------------------------------------------------------
// Bytes sh .. sh+15 of the 32-byte window (x, y), sh in [0, 15].
__device__ __forceinline__ uint4 window16(const uint4 x, const uint4 y, uint32_t sh) {
  // branch-free: move the window by 8 bytes, then by 4, then funnel-shift
  // the remaining 0..3 bytes (lanes with different shifts do not diverge)
  const bool h8 = (sh & 8u) != 0u, h4 = (sh & 4u) != 0u;
  const uint32_t b0 = h8 ? x.z : x.x, b1 = h8 ? x.w : x.y, b2 = h8 ? y.x : x.z;
  const uint32_t b3 = h8 ? y.y : x.w, b4 = h8 ? y.z : y.x, b5 = h8 ? y.w : y.y;
  const uint32_t a0 = h4 ? b1 : b0, a1 = h4 ? b2 : b1, a2 = h4 ? b3 : b2;
  const uint32_t a3 = h4 ? b4 : b3, a4 = h4 ? b5 : b4;
  const uint32_t b = (sh & 3u) * 8u;
  uint4 r;
  r.x = __funnelshift_r(a0, a1, b);
  r.y = __funnelshift_r(a1, a2, b);
  r.z = __funnelshift_r(a2, a3, b);
  r.w = __funnelshift_r(a3, a4, b);
  return r;
}

// v with its bytes from position b (0..16) on replaced by those of u
__device__ __forceinline__ uint32_t keep_low(uint32_t v, uint32_t u, int b) {
  const int c = b < 0 ? 0 : (b > 4 ? 4 : b);
  const uint32_t m = (uint32_t)((1ull << (8 * c)) - 1ull);
  return (v & m) | (u & ~m);
}
__device__ __forceinline__ uint4 take_from(const uint4 v, const uint4 u, uint32_t b) {
  const int bi = (int)b;
  return make_uint4(keep_low(v.x, u.x, bi), keep_low(v.y, u.y, bi - 4), keep_low(v.z, u.z, bi - 8),
                    keep_low(v.w, u.w, bi - 12));
}

__device__ __forceinline__ uint4 shfl_down4(const uint4 v, int d) {
  return make_uint4(__shfl_down_sync(0xffffffffu, v.x, d), __shfl_down_sync(0xffffffffu, v.y, d),
                    __shfl_down_sync(0xffffffffu, v.z, d), __shfl_down_sync(0xffffffffu, v.w, d));
}
__device__ __forceinline__ uint4 shfl_idx4(const uint4 v, int l) {
  return make_uint4(__shfl_sync(0xffffffffu, v.x, l), __shfl_sync(0xffffffffu, v.y, l),
                    __shfl_sync(0xffffffffu, v.z, l), __shfl_sync(0xffffffffu, v.w, l));
}

constexpr int CP_UNROLL = 4;   // groups of 32 words in flight per warp

// One warp copies `len` bytes from src to dst (both any alignment).  Whole
// destination words are written with 16-byte stores, each lane's word built
// from its own aligned source block and its right neighbour's (shuffled in,
// or loaded by the lane at a group's edge); the partial first and last words
// are written byte by byte, so the bytes of neighbouring pieces are never
// touched.  Every block read holds at least one byte of the source range.
// (Used for chunks whose pieces do not fit the shared-memory stage.)
__device__ __forceinline__ void warp_copy(uint8_t* dst, const uint8_t* src, uint64_t len, int lane) {
  const uint64_t d = (uint64_t)(uintptr_t)dst, d_end = d + len;
  const uint64_t head_end = ((d + 15) & ~15ull) < d_end ? ((d + 15) & ~15ull) : d_end;
  if ((uint64_t)lane < head_end - d) dst[lane] = __ldg(src + lane);
  if (head_end == d_end) return;
  const uint64_t full_lo = head_end, full_hi = d_end & ~15ull;
  if (full_hi > full_lo) {
    const uint64_t nw = (full_hi - full_lo) >> 4;
    const uint8_t* s_full = src + (full_lo - d);
    const uint32_t sig = (uint32_t)((uintptr_t)s_full & 15u);
    const uint4* A0 = reinterpret_cast<const uint4*>((uintptr_t)s_full & ~(uintptr_t)15);
    uint4* D0 = reinterpret_cast<uint4*>((uintptr_t)full_lo);
    for (uint64_t g0 = 0; g0 < nw; g0 += 32 * CP_UNROLL) {
      uint4 x[CP_UNROLL], y[CP_UNROLL];
#pragma unroll
      for (int u = 0; u < CP_UNROLL; ++u) {
        const uint64_t k = g0 + (uint64_t)u * 32 + lane;
        x[u] = make_uint4(0u, 0u, 0u, 0u);
        y[u] = x[u];
        if (k < nw) {
          x[u] = __ldg(A0 + k);
          const bool edge = (lane == 31 && (u == CP_UNROLL - 1 || k + 1 >= nw)) || k + 1 >= nw;
          if (sig && edge) y[u] = __ldg(A0 + k + 1);
        }
      }
      if (sig) {
#pragma unroll
        for (int u = 0; u < CP_UNROLL; ++u) {
          const uint64_t k = g0 + (uint64_t)u * 32 + lane;
          const uint4 nb = shfl_down4(x[u], 1);
          const uint4 nx = (u + 1 < CP_UNROLL) ? shfl_idx4(x[(u + 1) % CP_UNROLL], 0) : nb;
          const bool edge = (lane == 31 && (u == CP_UNROLL - 1 || k + 1 >= nw)) || k + 1 >= nw;
          if (!edge) y[u] = (lane == 31) ? nx : nb;
        }
      }
#pragma unroll
      for (int u = 0; u < CP_UNROLL; ++u) {
        const uint64_t k = g0 + (uint64_t)u * 32 + lane;
        if (k < nw) D0[k] = sig ? window16(x[u], y[u], sig) : x[u];
      }
    }
  }
  const uint64_t tail_lo = full_hi > head_end ? full_hi : head_end;
  if ((uint64_t)lane < d_end - tail_lo) dst[(tail_lo - d) + lane] = __ldg(src + (tail_lo - d) + lane);
}

// ---- TMA staging --------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_fence_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(parity)
      : "memory");
  return ok != 0u;
}
// The same wait, but the thread may sleep until the phase completes (or
// about `ns` nanoseconds pass) instead of returning at once.
__device__ __forceinline__ bool mbar_try_wait_sleep(uint64_t* bar, uint32_t parity, uint32_t ns) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(parity), "r"(ns)
      : "memory");
  return ok != 0u;
}
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
// bulk copy of `bytes` (multiple of 16) from 16-byte aligned global memory
// into 16-byte aligned shared memory, completing on `bar`
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_addr(dst)),
      "l"(src), "r"(bytes), "r"(smem_addr(bar))
      : "memory");
}

// tx bytes the current phase of `bar` waits for, without arriving
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.expect_tx.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes) : "memory");
}
// 16 bytes from 16-byte aligned global to 16-byte aligned shared memory,
// asynchronously (no register staging)
__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_addr(dst)), "l"(src) : "memory");
}
// the current phase of `bar` also waits for this thread's cp.async copies
// issued so far (the pending count goes up now and down when they land)
__device__ __forceinline__ void cp_async_track(uint64_t* bar) {
  asm volatile("cp.async.mbarrier.arrive.shared::cta.b64 [%0];" ::"r"(smem_addr(bar)) : "memory");
}

// Bounded wait on a stage barrier for the phase of parity `parity`; false
// (recording ERR_TIMEOUT and raising the CTA's abort flag) if it gave up or
// another warp of the CTA already did.  Called by every lane of a warp; the
// answer is the same for the whole warp (false if any lane gave up), so the
// warp's collective operations after it never see a split warp.
__device__ __forceinline__ bool stage_wait_lane(uint64_t* bar, uint32_t parity, uint32_t* err,
                                                volatile uint32_t* abort);
__device__ __forceinline__ bool stage_wait2(uint64_t* bar, uint32_t parity, uint32_t* err,
                                            volatile uint32_t* abort) {
  return __all_sync(0xffffffffu, stage_wait_lane(bar, parity, err, abort));
}
__device__ __forceinline__ bool stage_wait_lane(uint64_t* bar, uint32_t parity, uint32_t* err,
                                                volatile uint32_t* abort) {
  // at most 2^20 polls of up to ~1 us each
  for (uint32_t i = 0; i < (1u << 20); ++i) {
    if (mbar_try_wait_sleep(bar, parity, 1000u)) return true;
    if ((i & 255u) == 255u && (*abort || (ld_acquire(err) & ERR_TIMEOUT))) {
      *abort = 1u;
      return false;
    }
  }
  atomicOr(err, ERR_TIMEOUT);
  *abort = 1u;
  return false;
}

// One pipeline stage: the source bytes of one 16 KB output chunk, laid out
// piece by piece (each piece = the part of one member inside the chunk, read
// as the aligned 16-byte blocks that hold it).  Offsets inside the chunk are
// taken from wbase, the aligned word at or before the chunk's first byte.
struct CopyStage {
  uint32_t np;                    // pieces staged, or AC_FALLBACK
  uint32_t vbeg, vend;            // the chunk's bytes, relative to wbase
  uint32_t pad;
  unsigned long long wbase;       // absolute address of the chunk's first word
  unsigned long long rel_s, rel_e;   // the chunk's bytes, relative to the call's output
  unsigned long long j_lo;        // first member of the chunk
  // output start of each piece (+ end), relative to wbase (< 16400), and the
  // buffer offset of output byte wbase per piece (-16400 .. 24592)
  uint16_t pstart[AC_PIECES + 1];
  int16_t qbase[AC_PIECES];
  uint32_t pad2[3];
  // the 16 bytes before buf (the end of qbase) may be read and ignored: a
  // piece's first word can start before the piece's first staged block
  __align__(16) unsigned char buf[AC_BUF + 32];
};
constexpr uint32_t AC_FALLBACK = 0xFFFFFFFFu;
constexpr uint32_t AC_DONE = 0xFFFFFFFEu;      // no chunk: the consumers stop at this stage

size_t asm_copy_smem() { return AC_STAGES * sizeof(CopyStage); }

struct CopyCtx {
  const AssembleArgs* a;
  const uint64_t* cpos;
  const uint64_t* csrc;
  const uint32_t* ctfp;   // chunk table, or NULL (search instead)
  uint64_t out_base;      // absolute address of the call's first output byte
  uint64_t S, Mnz, n_chunks;
};

__device__ __forceinline__ uint64_t cpos_at(const CopyCtx& c, uint64_t j) {
  return j < c.Mnz ? c.cpos[j] : c.S;
}

// Largest j in [0, n) with pos[j] <= x (pos[0] = 0 <= x): 32 probes a round.
__device__ __forceinline__ uint64_t warp_search(const uint64_t* pos, uint64_t n, uint64_t x, int lane) {
  uint64_t lo = 0, hi = n;
  while (hi - lo > 1) {
    const uint64_t step = (hi - lo + 31) / 32;
    const uint64_t probe = lo + step * (uint64_t)lane;
    const bool le = probe < hi && pos[probe] <= x;
    const unsigned m = __ballot_sync(0xffffffffu, le);
    const uint64_t last = (uint64_t)(31 - __clz((int)m));
    lo = lo + step * last;
    hi = (lo + step < hi) ? lo + step : hi;
  }
  return lo;
}

// A producer warp stages chunk k: finds its members, builds the piece table
// and issues one bulk copy per piece, completing on `bar`.
__device__ void stage_chunk(const CopyCtx& c, uint64_t k, CopyStage* st, uint64_t* bar, int lane) {
  const uint64_t rs = k * AC_CHUNK;
  const uint64_t re = (rs + AC_CHUNK < c.S) ? rs + AC_CHUNK : c.S;
  uint64_t j_lo, j_hi;
  if (c.ctfp) {
    j_lo = c.ctfp[k];
    j_hi = (k + 1 < c.n_chunks) ? c.ctfp[k + 1] : c.Mnz - 1;
  } else {
    j_lo = warp_search(c.cpos, c.Mnz, rs, lane);
    j_hi = warp_search(c.cpos, c.Mnz, re - 1, lane);
  }
  const uint64_t np = j_hi - j_lo + 1;
  const uint64_t wbase = (c.out_base + rs) & ~15ull;
  if (lane == 0) {
    st->wbase = wbase;
    st->rel_s = rs;
    st->rel_e = re;
    st->j_lo = j_lo;
    st->vbeg = (uint32_t)(c.out_base + rs - wbase);
    st->vend = (uint32_t)(c.out_base + re - wbase);
  }
  const uint64_t arena = (uint64_t)(uintptr_t)c.a->arena;
  // a host-resident arena is read by the consumers with plain loads instead
  // of being staged; so is a chunk whose aligned blocks do not fit AC_BUF
  const bool tabled = np <= AC_PIECES && !c.a->arena_host;
  uint32_t roff = 0;   // running buffer offset (warp-uniform)
  uint32_t tx = 0;     // bytes of the pieces staged by bulk copies (per lane)
  if (tabled) {
    constexpr int R = 4;   // rounds of 32 pieces whose loads go out together
    for (uint64_t g0 = 0; g0 < np; g0 += 32 * R) {
      uint64_t p0[R], p1[R], cs[R];
#pragma unroll
      for (int u = 0; u < R; ++u) {
        const uint64_t i = g0 + (uint64_t)u * 32 + lane;
        p0[u] = p1[u] = cs[u] = 0;
        if (i < np) {
          const uint64_t j = j_lo + i;
          p0[u] = c.cpos[j];
          p1[u] = cpos_at(c, j + 1);
          cs[u] = c.csrc[j];
        }
      }
#pragma unroll
      for (int u = 0; u < R; ++u) {
        const uint64_t i = g0 + (uint64_t)u * 32 + lane;
        uint32_t size = 0, sh = 0, ps = 0;
        if (i < np) {
          const uint64_t ob = p0[u] > rs ? p0[u] : rs, oe = p1[u] < re ? p1[u] : re;
          const uint64_t src = arena + cs[u] + (ob - p0[u]);
          const uint64_t a0 = src & ~15ull, a1 = (src + (oe - ob) + 15) & ~15ull;
          size = (uint32_t)(a1 - a0);
          sh = (uint32_t)(src & 15u);
          ps = (uint32_t)(c.out_base + ob - wbase);
          if (size > AC_SMALL) tx += size;
        }
        uint32_t inc = size;
#pragma unroll
        for (int d = 1; d < 32; d <<= 1) {
          const uint32_t t = __shfl_up_sync(0xffffffffu, inc, d);
          if (lane >= d) inc += t;
        }
        const uint32_t my_off = roff + inc - size;
        if (i < np) {
          st->pstart[i] = (uint16_t)ps;
          st->qbase[i] = (int16_t)((int32_t)(my_off + sh) - (int32_t)ps);
        }
        roff += __shfl_sync(0xffffffffu, inc, 31);
      }
    }
  }
  const bool fits = tabled && roff <= AC_BUF;
  if (!fits) {
    if (lane == 0) {
      st->np = AC_FALLBACK;
      mbar_arrive(bar);   // completes the phase; consumers copy from global
    }
    __syncwarp();
    return;
  }
  // the stage completes when the bulk copies' bytes have landed, every
  // lane's cp.async copies of small pieces too, and lane 0 has arrived
  for (int d = 16; d > 0; d >>= 1) tx += __shfl_xor_sync(0xffffffffu, tx, d);
  if (lane == 0) {
    st->np = (uint32_t)np;
    st->pstart[np] = (uint16_t)(c.out_base + re - wbase);
    mbar_expect_tx(bar, tx);
  }
  __syncwarp();
  fence_proxy_async_smem();   // earlier generic accesses of this stage before async writes
  bool small = false;
  constexpr int R = 4;
  for (uint64_t i0 = lane; i0 < np; i0 += 32 * R) {
    uint64_t p0[R], cs[R];
#pragma unroll
    for (int u = 0; u < R; ++u) {
      const uint64_t i = i0 + (uint64_t)u * 32;
      p0[u] = cs[u] = 0;
      if (i < np) {
        p0[u] = c.cpos[j_lo + i];
        cs[u] = c.csrc[j_lo + i];
      }
    }
#pragma unroll
    for (int u = 0; u < R; ++u) {
      const uint64_t i = i0 + (uint64_t)u * 32;
      if (i >= np) break;
      const uint64_t ob = wbase + st->pstart[i] - c.out_base;      // relative
      const uint64_t oe = wbase + st->pstart[i + 1] - c.out_base;
      const uint64_t src = arena + cs[u] + (ob - p0[u]);
      const uint64_t a0 = src & ~15ull, a1 = (src + (oe - ob) + 15) & ~15ull;
      const uint32_t off = (uint32_t)(st->qbase[i] + (int32_t)st->pstart[i]) - (uint32_t)(src & 15u);
      const uint32_t size = (uint32_t)(a1 - a0);   // 0: a member that starts at the chunk's end
      if (size > AC_SMALL) {
        bulk_g2s(st->buf + off, reinterpret_cast<const void*>((uintptr_t)a0), size, bar);
      } else {
        // small pieces: one 16-byte asynchronous copy per block, no bulk copy
        for (uint32_t b = 0; b < size; b += 16)
          cp_async16(st->buf + off + b, reinterpret_cast<const void*>((uintptr_t)(a0 + b)));
        small = small || size != 0;
      }
    }
  }
  if (small) cp_async_track(bar);
  __syncwarp();
  if (lane == 0) mbar_arrive(bar);
}

// A chunk's pieces as a producer warp finds them.  With at most 32 pieces
// each lane keeps one piece's source block range in registers, so the
// chunk can be described (its global loads paid) before a stage is free and
// staged later without touching global memory again.
struct ChunkDesc {
  uint64_t k, rs, re, j_lo, np, wbase;
  bool inreg;                // np <= 32: the lane's piece below is valid if lane < np
  uint64_t a0;               // the lane's piece: first aligned source block
  uint32_t size, sh, ps;     // its staged bytes, source misalignment, output start (wbase-relative)
};

__device__ __forceinline__ void describe_chunk(const CopyCtx& c, uint64_t k, ChunkDesc& d, int lane) {
  d.k = k;
  d.rs = k * AC_CHUNK;
  d.re = (d.rs + AC_CHUNK < c.S) ? d.rs + AC_CHUNK : c.S;
  uint64_t j_hi;
  if (c.ctfp) {
    d.j_lo = c.ctfp[k];
    j_hi = (k + 1 < c.n_chunks) ? c.ctfp[k + 1] : c.Mnz - 1;
  } else {
    d.j_lo = warp_search(c.cpos, c.Mnz, d.rs, lane);
    j_hi = warp_search(c.cpos, c.Mnz, d.re - 1, lane);
  }
  d.np = j_hi - d.j_lo + 1;
  d.wbase = (c.out_base + d.rs) & ~15ull;
  d.inreg = d.np <= 32;
  d.a0 = 0;
  d.size = d.sh = d.ps = 0;
  if (d.inreg && (uint64_t)lane < d.np) {
    const uint64_t j = d.j_lo + lane;
    const uint64_t p0 = c.cpos[j], p1 = cpos_at(c, j + 1);
    const uint64_t ob = p0 > d.rs ? p0 : d.rs, oe = p1 < d.re ? p1 : d.re;
    const uint64_t src = (uint64_t)(uintptr_t)c.a->arena + c.csrc[j] + (ob - p0);
    d.a0 = src & ~15ull;
    d.size = (uint32_t)(((src + (oe - ob) + 15) & ~15ull) - d.a0);
    d.sh = (uint32_t)(src & 15u);
    d.ps = (uint32_t)(c.out_base + ob - d.wbase);
  }
}

// Stage a described chunk: piece table, expected bytes, one bulk copy per
// piece.  Chunks of more than 32 pieces take stage_chunk's general path.
__device__ void issue_chunk(const CopyCtx& c, const ChunkDesc& d, CopyStage* st, uint64_t* bar, int lane) {
  if (!d.inreg || c.a->arena_host) {
    stage_chunk(c, d.k, st, bar, lane);
    return;
  }
  uint32_t inc = d.size;
#pragma unroll
  for (int s = 1; s < 32; s <<= 1) {
    const uint32_t t = __shfl_up_sync(0xffffffffu, inc, s);
    if (lane >= s) inc += t;
  }
  const uint32_t my_off = inc - d.size;
  const uint32_t roff = __shfl_sync(0xffffffffu, inc, 31);
  if ((uint64_t)lane < d.np) {
    st->pstart[lane] = (uint16_t)d.ps;
    st->qbase[lane] = (int16_t)((int32_t)(my_off + d.sh) - (int32_t)d.ps);
  }
  if (lane == 0) {
    st->wbase = d.wbase;
    st->rel_s = d.rs;
    st->rel_e = d.re;
    st->j_lo = d.j_lo;
    st->vbeg = (uint32_t)(c.out_base + d.rs - d.wbase);
    st->vend = (uint32_t)(c.out_base + d.re - d.wbase);
    st->np = (uint32_t)d.np;
    st->pstart[d.np] = (uint16_t)(c.out_base + d.re - d.wbase);
  }
  __syncwarp();
  fence_proxy_async_smem();   // earlier generic accesses of this stage before async writes
  if (lane == 0) mbar_arrive_tx(bar, roff);
  __syncwarp();
  if ((uint64_t)lane < d.np && d.size)
    bulk_g2s(st->buf + my_off, reinterpret_cast<const void*>((uintptr_t)d.a0), d.size, bar);
}

__device__ __forceinline__ uint4 lds128(const unsigned char* p) {
  return *reinterpret_cast<const uint4*>(p);
}
// bytes A .. A+15 of the stage buffer (A may be down to -15)
__device__ __forceinline__ uint4 stage_word(const CopyStage* st, int32_t A) {
  const int32_t Aa = A & ~15;
  return window16(lds128(st->buf + Aa), lds128(st->buf + Aa + 16), (uint32_t)(A & 15));
}

// Consumer warp cw writes words [w0, w1) of a staged chunk, a lane per
// 16-byte word.  A word inside one piece is one shifted 16-byte read of the
// stage; a word that meets a piece boundary merges its pieces' bytes.  The
// chunk's first and last words may hold bytes of neighbouring chunks: only
// the chunk's own bytes of them are written, byte by byte.
__device__ void emit_range(const CopyStage* st, uint32_t cw, int lane) {
  const uint32_t np = st->np, vbeg = st->vbeg, vend = st->vend;
  const uint64_t wbase = st->wbase;
  const uint32_t nW = (vend + 15u) >> 4;
  const uint32_t w0 = (nW * cw) / AC_CONSUMERS, w1 = (nW * (cw + 1)) / AC_CONSUMERS;
  if (w0 >= w1) return;
  const uint32_t first = (w0 * 16u > vbeg) ? w0 * 16u : vbeg;
  uint32_t a = 0, b = np;   // the piece holding byte `first` (pstart[0] = vbeg)
  while (b - a > 1) {
    const uint32_t m = (a + b) >> 1;
    if (st->pstart[m] <= first) a = m; else b = m;
  }
  uint32_t icur = a;
#pragma unroll 1
  for (uint32_t g = w0; g < w1; g += 32) {
    const uint32_t w = g + (uint32_t)lane;
    uint32_t i = icur;
    if (w < w1) {
      const uint32_t wr = w * 16u;
      const uint32_t lo = wr > vbeg ? wr : vbeg;
      const uint32_t hi = (wr + 16u < vend) ? wr + 16u : vend;
      // the piece holding byte lo: the warp's last piece or the next (large
      // pieces), else a search of the rest (many small pieces per chunk)
      uint32_t pe = st->pstart[i + 1];
      if (pe <= lo) {
        ++i;
        pe = st->pstart[i + 1];
        if (pe <= lo) {
          uint32_t ia = i + 1, ib = np;   // pstart[ia] <= lo < pstart[np]
          while (ib - ia > 1) {
            const uint32_t m = (ia + ib) >> 1;
            if (st->pstart[m] <= lo) ia = m; else ib = m;
          }
          i = ia;
          pe = st->pstart[i + 1];
        }
      }
      // bytes [lo, pe) come from piece i; a word that reaches further takes
      // the rest from the following pieces, one boundary at a time
      uint4 v = stage_word(st, st->qbase[i] + (int32_t)wr);
      while (pe < hi) {
        ++i;
        v = take_from(v, stage_word(st, st->qbase[i] + (int32_t)wr), pe - wr);
        pe = st->pstart[i + 1];
      }
      uint4* dst = reinterpret_cast<uint4*>((uintptr_t)(wbase + wr));
      if (lo == wr && hi == wr + 16u) {
        *dst = v;
      } else {
        // the chunk's first or last word: only the chunk's own bytes
        const uint32_t vv[4] = {v.x, v.y, v.z, v.w};
        uint8_t* d8 = reinterpret_cast<uint8_t*>(dst);
#pragma unroll
        for (int t = 0; t < 16; ++t)
          if ((uint32_t)t >= lo - wr && (uint32_t)t < hi - wr) d8[t] = (uint8_t)(vv[t >> 2] >> (8 * (t & 3)));
      }
    }
    icur = __shfl_sync(0xffffffffu, i, 31);
  }
}

// A chunk whose pieces do not fit a stage: consumer warps copy slices of it
// straight from global memory.
__device__ void emit_direct(const CopyCtx& c, const CopyStage* st, uint32_t cw, int lane) {
  constexpr uint64_t SLICE = (AC_CHUNK + AC_CONSUMERS - 1) / AC_CONSUMERS;
  const uint64_t rs = st->rel_s, re = st->rel_e;
  uint64_t ra = rs + (uint64_t)cw * SLICE;
  const uint64_t rb = (ra + SLICE < re) ? ra + SLICE : re;
  if (ra >= rb) return;
  uint64_t k = warp_search(c.cpos, c.Mnz, ra, lane);
  for (; ra < rb; ++k) {
    const uint64_t pk = c.cpos[k], pn = cpos_at(c, k + 1);
    const uint64_t e = pn < rb ? pn : rb;
    warp_copy(c.a->out + (c.out_base - (uint64_t)(uintptr_t)c.a->out) + ra,
              c.a->arena + c.csrc[k] + (ra - pk), e - ra, lane);
    ra = e;
  }
}

// A copy of at most AC_SMALL_CHUNKS chunks is latency-bound: every warp of
// the participating CTAs takes 2 KB slices of the output in turn and copies
// the member pieces inside each straight from the arena (no claims, staging
// or barriers), the slice's first member found from the chunk table and one
// warp-wide probe of the next 32 members.
constexpr uint64_t AC_SLICE = 2048;
__device__ void copy_small(const CopyCtx& c, uint64_t gw, uint64_t n_w, int lane) {
  const uint64_t n_sl = ceil_div(c.S, AC_SLICE);
  for (uint64_t sl = gw; sl < n_sl; sl += n_w) {
    uint64_t ra = sl * AC_SLICE;
    const uint64_t rb = (ra + AC_SLICE < c.S) ? ra + AC_SLICE : c.S;
    uint64_t k;
    if (c.ctfp) {   // the member holding the chunk's first byte holds or precedes ra
      const uint64_t k0 = c.ctfp[ra / AC_CHUNK], probe = k0 + (uint64_t)lane;
      const unsigned m = __ballot_sync(0xffffffffu, probe < c.Mnz && c.cpos[probe] <= ra);
      k = (m == 0xffffffffu) ? warp_search(c.cpos, c.Mnz, ra, lane) : k0 + (uint64_t)(__popc(m) - 1);
    } else {
      k = warp_search(c.cpos, c.Mnz, ra, lane);
    }
    for (; ra < rb; ++k) {
      const uint64_t pk = c.cpos[k], pn = cpos_at(c, k + 1);
      const uint64_t e = pn < rb ? pn : rb;
      warp_copy(c.a->out + (c.out_base - (uint64_t)(uintptr_t)c.a->out) + ra,
                c.a->arena + c.csrc[k] + (ra - pk), e - ra, lane);
      ra = e;
    }
  }
}

// The copy: per-parent outputs, then the chunks of the call's output, each
// CTA taking every n_part-th chunk.  Warps 0..AC_PRODUCERS-1 stage chunks
// into a ring of AC_STAGES stages (producer p takes the CTA's chunks i with
// i % AC_PRODUCERS == p), the other warps write them out in order; full
// and empty mbarriers per stage hand the stages back and forth.
// Sized to leave room beside it: two CTAs per SM take 2 x 320 threads x 80
// registers and 2 x 3 stages of shared memory, so a planning CTA (56
// registers) of a later wave (another stream) can be resident on the same SM
// while a copy runs.
__global__ void __maxnreg__(80) asm_copy_kernel(AssembleArgs a) {
  wait_predecessor();
  extern __shared__ __align__(128) unsigned char ac_smem[];
  __shared__ __align__(8) uint64_t full_bar[AC_STAGES];
  __shared__ __align__(8) uint64_t empty_bar[AC_STAGES];
  __shared__ uint32_t s_issued[AC_STAGES];
  __shared__ uint32_t s_abort;
  __shared__ uint32_t s_round[2];   // the current and next claimed rounds (dynamic chunks)
  CopyStage* stages = reinterpret_cast<CopyStage*>(ac_smem);
  DevScalars* ds = a.ds;
  const PlanHdr hdr = *a.plan.hdr;
  const uint64_t n = hdr.n, S = hdr.bytes;
  const uint64_t base = a.cursor ? *a.cursor : 0ull;
  // conditions every CTA sees the same way
  bool failed = hdr.err != 0u;
  if (!failed && hdr.max_end > a.arena_bytes) {   // the arena passed here must hold what was accepted
    failed = true;
    if (threadIdx.x == 0) atomicOr(&ds->err, ERR_INVAL);
  }
  const bool too_many = !a.user_list && n > a.n_host;   // outputs hold fewer parents
  const bool too_big = base + S > a.out_cap;
  if (!failed && (too_many || too_big)) {
    failed = true;
    if (threadIdx.x == 0) atomicOr(&ds->err, ERR_CAPACITY);
  }
  CopyCtx c;
  c.a = &a;
  c.cpos = a.plan.cpos;
  c.csrc = a.plan.csrc;
  c.ctfp = hdr.chunks_ok ? a.plan.ctfp : nullptr;
  c.out_base = (uint64_t)(uintptr_t)a.out + base;
  c.S = S;
  c.Mnz = hdr.nnz;
  const uint64_t n_chunks = (!failed && S) ? ceil_div(S, AC_CHUNK) : 0;
  c.n_chunks = n_chunks;
  const uint64_t par_units = failed ? 0 : ceil_div(n + 1, (uint64_t)AC_THREADS * 8);
  uint64_t units = n_chunks > par_units ? n_chunks : par_units;
  if (units == 0) units = 1;   // one CTA still finishes the call
  const uint32_t n_part = participants(units);
  if (blockIdx.x >= n_part) return;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;

  if (!failed) {
    // per-parent outputs: status (commit plans), offsets, lengths, and the
    // list structure's entry offsets made absolute
    {
      const uint64_t stride = (uint64_t)n_part * blockDim.x;
      const uint64_t gt0 = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
      if (a.elem_base)
        for (uint64_t g = gt0; g < hdr.M; g += stride) a.elem_off[g] += base;
      for (uint64_t i = gt0; i <= n; i += stride) {
        const uint64_t o = a.plan.off[i];
        a.out_off[i] = base + o;
        if (i == n) break;
        if (!a.user_list) a.status[i] = a.list.status[i];   // a caller's list has them already
        if (a.out_len) {
          const uint64_t len = a.plan.off[i + 1] - o;
          if (len > 0xFFFFFFFFull) atomicOr(&ds->err, ERR_OVERFLOW);
          a.out_len[i] = (uint32_t)len;
        }
      }
    }
    if (n_chunks <= a.small_chunks) {
      copy_small(c, (uint64_t)blockIdx.x * (AC_THREADS / 32) + warp, (uint64_t)n_part * (AC_THREADS / 32),
                 lane);
    } else {
    if (threadIdx.x == 0) {
      for (int s = 0; s < AC_STAGES; ++s) {
        mbar_init(&full_bar[s], 1);
        mbar_init(&empty_bar[s], AC_CONSUMERS);
        s_issued[s] = 0u;
      }
      s_abort = 0u;
      mbar_fence_init();
    }
    __syncthreads();
    volatile uint32_t* abort = &s_abort;
#if RO_COPY_DYNAMIC
    if (warp < AC_PRODUCERS) {
      // Chunks are claimed in rounds of AC_PRODUCERS from a counter the grid
      // shares, so a CTA that starts late (its SM busy with another stream's
      // work) takes fewer: producer 0 claims the next round while this one
      // is staged and hands each round to the other producer at a named
      // barrier; stage index AC_PRODUCERS * r + warp holds chunk base_r +
      // warp.  Both producers leave at the same round (the barrier needs
      // both), and the first stage index left unfilled is marked done for
      // the consumers.
      ChunkDesc d;
      uint32_t next = 0;
      if (warp == 0 && lane == 0) next = atomicAdd(&ds->tile_ctr[TS_ASM_COPY], (uint32_t)AC_PRODUCERS);
      uint32_t r = 0;
      for (;; ++r) {
        if (warp == 0 && lane == 0) {
          // a wait that gave up stops both producers at the same round
          s_round[r & 1u] = *abort ? 0xFFFFFFFFu : next;
          if ((uint64_t)next < n_chunks)   // the claim of the following round, ahead
            next = atomicAdd(&ds->tile_ctr[TS_ASM_COPY], (uint32_t)AC_PRODUCERS);
        }
        asm volatile("bar.sync 1, %0;" ::"r"(AC_PRODUCERS * 32) : "memory");
        const uint64_t base_r = s_round[r & 1u];
        if (base_r >= n_chunks) break;
        const uint64_t k = base_r + (uint64_t)warp;
        const uint32_t i = AC_PRODUCERS * r + (uint32_t)warp;
        const uint32_t s = i % AC_STAGES, u = i / AC_STAGES;
        if (k < n_chunks) describe_chunk(c, k, d, lane);
        if (u > 0 && !stage_wait2(&empty_bar[s], (u - 1u) & 1u, &ds->err, abort)) continue;
        if (k < n_chunks) {
          issue_chunk(c, d, &stages[s], &full_bar[s], lane);
        } else if (lane == 0) {   // the last round is short: the consumers stop here
          stages[s].np = AC_DONE;
          mbar_arrive(&full_bar[s]);
        }
        if (lane == 0) s_issued[s] = u + 1u;
        __syncwarp();
      }
      const bool aborted = __any_sync(0xffffffffu, *abort != 0u);
      if (warp == 0 && !aborted) {   // the first stage index left unfilled
        const uint32_t i = AC_PRODUCERS * r;
        const uint32_t s = i % AC_STAGES, u = i / AC_STAGES;
        if (u == 0 || stage_wait2(&empty_bar[s], (u - 1u) & 1u, &ds->err, abort)) {
          if (lane == 0) {
            stages[s].np = AC_DONE;
            mbar_arrive(&full_bar[s]);
            s_issued[s] = u + 1u;
          }
        }
        __syncwarp();
      }
      // this lane's cp.async copies of small pieces land before the CTA can
      // exit (on an abort nobody else waits for them)
      asm volatile("cp.async.wait_all;" ::: "memory");
    } else {
      const uint32_t cw = (uint32_t)(warp - AC_PRODUCERS);
      for (uint32_t i = 0;; ++i) {
        const uint32_t s = i % AC_STAGES, u = i / AC_STAGES;
        if (!stage_wait2(&full_bar[s], u & 1u, &ds->err, abort)) break;
        const uint32_t np = stages[s].np;
        if (np == AC_DONE) break;
        if (np == AC_FALLBACK)
          emit_direct(c, &stages[s], cw, lane);
        else
          emit_range(&stages[s], cw, lane);
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty_bar[s]);
      }
    }
#else
    if (warp < AC_PRODUCERS) {
      // each chunk is described before its stage frees up: the loads of
      // chunk i+AC_PRODUCERS overlap the copies and the writing of chunk i
      ChunkDesc d;
      uint32_t i = (uint32_t)warp;
      uint64_t k = blockIdx.x + (uint64_t)i * n_part;
      if (k < n_chunks) describe_chunk(c, k, d, lane);
      while (k < n_chunks) {
        const uint32_t s = i % AC_STAGES, u = i / AC_STAGES;
        if (u > 0 && !stage_wait2(&empty_bar[s], (u - 1u) & 1u, &ds->err, abort)) break;
        issue_chunk(c, d, &stages[s], &full_bar[s], lane);
        if (lane == 0) s_issued[s] = u + 1u;
        i += AC_PRODUCERS;
        k = blockIdx.x + (uint64_t)i * n_part;
        if (k < n_chunks) describe_chunk(c, k, d, lane);
      }
      // this lane's cp.async copies of small pieces land before the CTA can
      // exit (on an abort nobody else waits for them)
      asm volatile("cp.async.wait_all;" ::: "memory");
    } else {
      const uint32_t cw = (uint32_t)(warp - AC_PRODUCERS);
      for (uint32_t i = 0;; ++i) {
        const uint64_t k = blockIdx.x + (uint64_t)i * n_part;
        if (k >= n_chunks) break;
        const uint32_t s = i % AC_STAGES, u = i / AC_STAGES;
        if (!stage_wait2(&full_bar[s], u & 1u, &ds->err, abort)) break;
        if (stages[s].np == AC_FALLBACK)
          emit_direct(c, &stages[s], cw, lane);
        else
          emit_range(&stages[s], cw, lane);
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty_bar[s]);
      }
    }
#endif
    __syncthreads();
    // a wait that gave up: give the copies still in flight a bounded chance
    // to land before the CTA's shared memory is released
    if (s_abort && threadIdx.x == 0) {
      for (int s = 0; s < AC_STAGES; ++s) {
        if (!s_issued[s]) continue;
        bool landed = false;
        for (uint32_t t = 0; t < (1u << 20) && !landed; ++t)
          landed = mbar_try_wait(&full_bar[s], (s_issued[s] - 1u) & 1u);
        // bulk copies still in flight as the CTA exits: recorded apart
        if (!landed) atomicOr(&ds->err, ERR_DRAIN);
      }
    }
    }
  }
  // this CTA's bytes are done: the next copy on the stream may be scheduled
  // into the space it leaves (it waits for this grid before it reads anything)
  allow_successor();
  if (threadIdx.x == 0) {
    if (ticket(&ds->exit_ctr[TS_ASM_COPY]) == n_part - 1) {
      if (!failed && a.cursor) *a.cursor = base + S;
      if (!failed && hdr.incomplete) ds->stats[6] += hdr.incomplete;
      if (a.out_bytes) *a.out_bytes = S;
      if (a.n_elems_out) *a.n_elems_out = hdr.M;
      ds->as_bytes = S;
      ds->as_elems = hdr.M;
      a.plan.hdr->err = 0u;   // the plan is consumed
      ds->tile_ctr[TS_ASM_COPY] = 0u;   // the chunk counter, for the next copy
      ds->exit_ctr[TS_ASM_COPY] = 0u;
    }
  }
}

void launch_assemble_plan(const LaunchCfg& L, const AssembleArgs& a) {
  if (a.user_list) {
    const uint64_t tiles = ceil_div(a.n_host, (uint64_t)AP_THREADS * AP_ITEMS);
    const int grid = (int)std::max<uint64_t>(1, std::min<uint64_t>(tiles, (uint64_t)L.grid_aparents));
    launch_k(L, K_APARENTS, asm_parents_kernel, grid, AP_THREADS, 0, a);
  }
  launch_k(L, K_AMEMBERS, asm_members_kernel, L.grid_amembers, AM_THREADS, 0, a);
}

void launch_assemble_copy(const LaunchCfg& L, const AssembleArgs& a) {
  launch_k(L, K_ACOPY, asm_copy_kernel, L.grid_acopy, AC_THREADS, asm_copy_smem(), a);
}

// opt in to the copy kernel's dynamic shared memory (AC_STAGES pipeline stages)
cudaError_t prepare_assemble_kernels() {
  return cudaFuncSetAttribute(asm_copy_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)asm_copy_smem());
}

// F.filter (Table 3) on a report batch: Present with a false mask -> Dropped
__global__ void filter_kernel(uint8_t* state, const uint8_t* keep, uint64_t n) {
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  for (uint64_t r = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; r < n; r += stride)
    if (state[r] == ST_PRESENT && !keep[r]) state[r] = ST_DROPPED;
}

void launch_filter(cudaStream_t s, uint8_t* state, const uint8_t* keep, uint64_t n, int grid) {
  const uint64_t need = ceil_div(n, 256);
  const int g = (int)(need < (uint64_t)grid ? (need ? need : 1) : grid);
  filter_kernel<<<g, 256, 0, s>>>(state, keep, n);
}

const void* kernel_ptr_assemble(int which) {
  if (which == K_APARENTS) return (const void*)asm_parents_kernel;
  if (which == K_AMEMBERS) return (const void*)asm_members_kernel;
  return (const void*)asm_copy_kernel;
}

}  // namespace ro
