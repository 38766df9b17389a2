// k_assemble.cu — ro_assemble kernels (Section 4.2, Reduce).
//
// A completed parent is Suppressed if a member Failed or was Suppressed,
// otherwise Present with the Present members' payloads concatenated by
// ordinal (Dropped members add nothing).  The work is a segmented byte gather
// from the result arena, done in three passes:
//   asm_parents  per listed parent: outcome, number of members to gather
//                (0 unless Present), exclusive scan of those counts (member
//                bases), and for every 2048-member tile the parent that
//                contains its first member.
//   asm_members  per member (load-balanced over tiles of 2048 members, so a
//                100k-member parent is spread over many CTAs): read its
//                record, scan the Present bytes (single-pass look-back) and
//                emit, for every member that contributes bytes, its output
//                position and arena offset, plus each parent's output offset
//                and, for every 16 KB output chunk, the first member in it.
//   asm_copy     per 16 KB output chunk: stage the chunk's members in shared
//                memory and write the chunk as aligned 16-byte stores.  Each
//                store takes its bytes from one member with two aligned
//                16-byte loads and a funnel shift (source and destination
//                alignments differ arbitrarily); words that straddle members
//                or the ends of the output are assembled byte by byte.
#include <algorithm>

#include "ro_internal.h"

namespace ro {

constexpr int TS_ASM_COPY = 5;

__device__ __forceinline__ uint64_t asm_list_count(const AssembleArgs& a, bool* over) {
  uint64_t n;
  if (a.list_is_commit)
    n = a.ds->cm_n_done;
  else if (a.d_n)
    n = *a.d_n;
  else
    n = a.n_host;
  *over = n > a.n_host;
  return n > a.n_host ? a.n_host : n;
}

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
__global__ void __launch_bounds__(AP_THREADS) asm_parents_kernel(AssembleArgs a) {
  __shared__ unsigned long long s_scan[33];
  __shared__ uint32_t s_tile;
  __shared__ unsigned long long s_prefix;
  __shared__ unsigned long long s_incomplete;
  DevScalars* ds = a.ds;
  bool over = false;
  const uint64_t n = asm_list_count(a, &over);
  if (over) {
    if (threadIdx.x == 0) {
      ds->as_err = 1u;
      atomicOr(&ds->err, ERR_CAPACITY);
    }
    return;   // no tile claimed
  }
  if (threadIdx.x == 0) s_incomplete = 0;
  const uint64_t TILE = (uint64_t)AP_THREADS * AP_ITEMS;
  const uint64_t n_tiles = ceil_div(n, TILE);
  for (;;) {
    if (threadIdx.x == 0) s_tile = claim_tile(&ds->tile_ctr[TS_ASM_PARENTS]);
    __syncthreads();
    const uint32_t tile = s_tile;
    __syncthreads();
    if (tile >= n_tiles) break;
    const uint64_t i0 = tile * TILE + (uint64_t)threadIdx.x * AP_ITEMS;
    uint32_t m[AP_ITEMS];
    unsigned long long mine = 0;
    uint32_t incomplete = 0;
#pragma unroll
    for (int k = 0; k < AP_ITEMS; ++k) {
      const uint64_t i = i0 + k;
      m[k] = 0;
      if (i >= n) continue;
      const uint64_t p = a.list[i];
      uint8_t st = ST_PENDING;
      if (p < a.P) {
        const unsigned long long v = a.pw[p];
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
      a.status[i] = st;
      mine += m[k];
    }
    if (incomplete) atomicAdd(&s_incomplete, (unsigned long long)incomplete);
    unsigned long long total;
    unsigned long long excl = block_excl_scan(mine, s_scan, &total);
    if (threadIdx.x == 0) s_prefix = lookback_exclusive(a.ts_parents, tile, total, ds->epoch[TS_ASM_PARENTS], &ds->err);
    __syncthreads();
    unsigned long long run = s_prefix + excl;
#pragma unroll
    for (int k = 0; k < AP_ITEMS; ++k) {
      const uint64_t i = i0 + k;
      if (i >= n) break;
      a.mb[i] = (uint32_t)run;
      if (m[k]) {
        for (uint64_t b = ceil_div(run, AM_TILE); b * AM_TILE < run + m[k] && b < a.mtfp_cap; ++b)
          a.mtfp[b] = (uint32_t)i;
      }
      run += m[k];
    }
    if (tile == n_tiles - 1 && threadIdx.x == AP_THREADS - 1) {
      a.mb[n] = (uint32_t)run;
      ds->as_M = run;
      ds->as_n = n;
      if (run > a.member_cap) {
        ds->as_err = 1u;
        atomicOr(&ds->err, ERR_CAPACITY);
      }
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    if (s_incomplete) atomicAdd(&ds->stats[6], s_incomplete);
    if (n_tiles == 0 && blockIdx.x == 0) {
      a.mb[0] = 0;
      ds->as_M = 0;
      ds->as_n = 0;
    }
    retire_cta(ds, TS_ASM_PARENTS);
  }
}

// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(AM_THREADS) asm_members_kernel(AssembleArgs a) {
  __shared__ uint32_t s_mb[AM_SMEM_CAP];
  __shared__ uint32_t s_coff[AM_SMEM_CAP];
  __shared__ Pair64 s_scan[33];
  __shared__ uint32_t s_tile;
  __shared__ Pair64 s_prefix;
  DevScalars* ds = a.ds;
  if (ds->as_err) return;   // nothing claimed
  const uint64_t n = ds->as_n, M = ds->as_M;
  const uint64_t base = a.cursor ? *a.cursor : 0ull;
  const uint64_t out_addr = (uint64_t)(uintptr_t)a.out;
  const uint64_t origin = (out_addr + base) & ~15ull;
  const uint64_t n_tiles = ceil_div(M, AM_TILE);

  if (M == 0) {
    if (blockIdx.x == 0) {
      for (uint64_t i = threadIdx.x; i <= n; i += blockDim.x) a.out_off[i] = base;
      if (threadIdx.x == 0) {
        ds->as_bytes = 0;
        ds->as_Mnz = 0;
        ds->as_base = base;
        if (base > a.out_cap) {
          ds->as_err = 1u;
          atomicOr(&ds->err, ERR_CAPACITY);
        }
      }
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
    const uint64_t i_lo = a.mtfp[tile];
    const uint64_t i_hi = (tile + 1 < n_tiles) ? a.mtfp[tile + 1] : n - 1;
    const uint64_t R = i_hi - i_lo + 1;
    const bool staged = R <= AM_SMEM_CAP;
    if (staged) {
      for (uint64_t k = threadIdx.x; k < R; k += blockDim.x) {
        s_mb[k] = a.mb[i_lo + k];
        const uint64_t p = a.list[i_lo + k];   // listed ids may name no parent
        s_coff[k] = p < a.P ? (uint32_t)a.offsets[p] : 0u;
      }
    }
    __syncthreads();

    const uint64_t gt = g0 + (uint64_t)threadIdx.x * AM_ITEMS;
    uint32_t contrib[AM_ITEMS];
    uint64_t src[AM_ITEMS];
    uint32_t par[AM_ITEMS];
    bool first[AM_ITEMS];
    Pair64 mine{0, 0};
#pragma unroll
    for (int k = 0; k < AM_ITEMS; ++k) {
      const uint64_t g = gt + k;
      contrib[k] = 0;
      src[k] = 0;
      par[k] = 0;
      first[k] = false;
      if (g >= M) continue;
      uint64_t i, mbi, coff;
      if (staged) {
        const uint32_t kk = last_le_u(s_mb, 0u, (uint32_t)R, g);
        i = i_lo + kk;
        mbi = s_mb[kk];
        coff = s_coff[kk];
      } else {
        uint64_t lo = i_lo, hi = i_hi + 1;
        while (hi - lo > 1) {
          const uint64_t mid = lo + ((hi - lo) >> 1);
          if (a.mb[mid] <= g)
            lo = mid;
          else
            hi = mid;
        }
        i = lo;
        mbi = a.mb[lo];
        coff = a.offsets[a.list[lo]];
      }
      const Rec r = a.rec[coff + (g - mbi)];
      if (w_state(r.w) == ST_PRESENT && r.len) {
        contrib[k] = r.len;
        src[k] = w_off(r.w);
        // the arena passed here must hold what the commit accepted
        if (src[k] > a.arena_bytes || (uint64_t)r.len > a.arena_bytes - src[k]) {
          atomicOr(&ds->err, ERR_INVAL);
          ds->as_err = 1u;
        }
      }
      par[k] = (uint32_t)i;
      first[k] = (g == mbi);
      mine.a += contrib[k];
      mine.b += contrib[k] ? 1ull : 0ull;
    }
    Pair64 total;
    Pair64 excl = block_excl_scan_pair(mine, s_scan, &total);
    if (threadIdx.x == 0)
      s_prefix = lookback_exclusive(a.ts_members, tile, total, ds->epoch[TS_ASM_MEMBERS], &ds->err);
    __syncthreads();
    Pair64 run = s_prefix + excl;   // (bytes, contributing members) before my first item
#pragma unroll
    for (int k = 0; k < AM_ITEMS; ++k) {
      const uint64_t g = gt + k;
      if (g >= M) break;
      const uint64_t pos = base + run.a;
      if (first[k]) {
        // the parent starts here, and so do the member-less parents listed just before it
        a.out_off[par[k]] = pos;
        for (int64_t q = (int64_t)par[k] - 1; q >= 0; --q) {
          const uint32_t mbq = (staged && (uint64_t)q >= i_lo) ? s_mb[q - i_lo] : a.mb[q];
          if (mbq != g) break;
          a.out_off[q] = pos;
        }
      }
      if (contrib[k]) {
        const uint64_t j = run.b;
        if (j < a.member_cap) {
          a.cpos[j] = pos;
          a.csrc[j] = src[k];
        }
        const uint64_t A = out_addr + pos, E = A + contrib[k];
        if (j == 0 && a.ctfp_cap) a.ctfp[0] = 0u;
        for (uint64_t b = ceil_div(A - origin, AC_CHUNK); origin + b * AC_CHUNK < E && b < a.ctfp_cap; ++b)
          a.ctfp[b] = (uint32_t)j;
        run.b += 1;
        run.a += contrib[k];
      }
    }
    if (tile == n_tiles - 1 && threadIdx.x == AM_THREADS - 1) {
      const uint64_t end = base + run.a;
      a.out_off[n] = end;
      for (int64_t q = (int64_t)n - 1; q >= 0; --q) {
        if ((uint64_t)a.mb[q] != M) break;   // member-less parents at the very end
        a.out_off[q] = end;
      }
      ds->as_bytes = run.a;
      ds->as_Mnz = run.b;
      ds->as_base = base;
      if (end > a.out_cap || ceil_div(out_addr + end - origin, AC_CHUNK) > a.ctfp_cap) {
        ds->as_err = 1u;
        atomicOr(&ds->err, ERR_CAPACITY);
      }
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) retire_cta(ds, TS_ASM_MEMBERS);
}

// ---------------------------------------------------------------------------
// 16 bytes starting at any address, from the one or two aligned 16-byte
// blocks that hold them (both lie inside the record being read).
__device__ __forceinline__ uint4 load16_any(const uint8_t* p) {
  const uintptr_t addr = (uintptr_t)p;
  const uint32_t sh = (uint32_t)(addr & 15u);
  const uint4* q = reinterpret_cast<const uint4*>(addr & ~(uintptr_t)15);
  const uint4 x = __ldg(q);
  if (sh == 0) return x;
  const uint4 y = __ldg(q + 1);
  const uint32_t b = (sh & 3u) * 8u;
  uint32_t a0, a1, a2, a3, a4;
  switch (sh >> 2) {
    case 0: a0 = x.x; a1 = x.y; a2 = x.z; a3 = x.w; a4 = y.x; break;
    case 1: a0 = x.y; a1 = x.z; a2 = x.w; a3 = y.x; a4 = y.y; break;
    case 2: a0 = x.z; a1 = x.w; a2 = y.x; a3 = y.y; a4 = y.z; break;
    default: a0 = x.w; a1 = y.x; a2 = y.y; a3 = y.z; a4 = y.w; break;
  }
  uint4 r;
  r.x = __funnelshift_r(a0, a1, b);
  r.y = __funnelshift_r(a1, a2, b);
  r.z = __funnelshift_r(a2, a3, b);
  r.w = __funnelshift_r(a3, a4, b);
  return r;
}

__global__ void __launch_bounds__(AC_THREADS) asm_copy_kernel(AssembleArgs a) {
  __shared__ uint64_t s_pos[AC_SMEM_CAP + 1];
  __shared__ uint64_t s_src[AC_SMEM_CAP];
  DevScalars* ds = a.ds;
  const bool failed = ds->as_err != 0u;
  const uint64_t n = ds->as_n, S = ds->as_bytes, Mnz = ds->as_Mnz, base = ds->as_base;
  const uint64_t out_addr = (uint64_t)(uintptr_t)a.out;

  if (!failed) {
    // per-parent byte counts
    if (a.out_len) {
      const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
      for (uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
        const uint64_t len = a.out_off[i + 1] - a.out_off[i];
        if (len > 0xFFFFFFFFull) atomicOr(&ds->err, ERR_OVERFLOW);
        a.out_len[i] = (uint32_t)len;
      }
    }
    const uint64_t start = out_addr + base, end = start + S;
    const uint64_t origin = start & ~15ull;
    const uint64_t n_chunks = S ? ceil_div(end - origin, AC_CHUNK) : 0;
    const uint64_t stop = (end + 15) & ~15ull;
    for (uint64_t b = blockIdx.x; b < n_chunks; b += gridDim.x) {
      const uint64_t cs = origin + b * AC_CHUNK;
      const uint64_t ce = (cs + AC_CHUNK < stop) ? cs + AC_CHUNK : stop;
      const uint64_t j_lo = a.ctfp[b];
      const uint64_t j_hi = (b + 1 < n_chunks) ? a.ctfp[b + 1] : Mnz - 1;
      const uint64_t Rm = j_hi - j_lo + 1;
      const bool staged = Rm + 1 <= AC_SMEM_CAP;
      const uint64_t end_rel = base + S;
      if (staged) {
        for (uint64_t k = threadIdx.x; k <= Rm; k += blockDim.x) {
          const uint64_t j = j_lo + k;
          s_pos[k] = (j < Mnz) ? a.cpos[j] : end_rel;
          if (k < Rm) s_src[k] = a.csrc[j];
        }
      }
      __syncthreads();
      // position (relative to out) where member j_lo + k starts; k == Rm: end
      auto pos_of = [&](uint64_t k) -> uint64_t {
        if (staged) return s_pos[k];
        const uint64_t j = j_lo + k;
        return (j < Mnz) ? a.cpos[j] : end_rel;
      };
      auto src_of = [&](uint64_t k) -> uint64_t { return staged ? s_src[k] : a.csrc[j_lo + k]; };
      auto find = [&](uint64_t rel) -> uint64_t {   // member holding relative byte rel
        uint64_t lo = 0, hi = Rm;
        while (hi - lo > 1) {
          const uint64_t mid = lo + ((hi - lo) >> 1);
          if (pos_of(mid) <= rel)
            lo = mid;
          else
            hi = mid;
        }
        return lo;
      };
      const uint64_t n_words = (ce - cs) >> 4;
      for (uint64_t wi = threadIdx.x; wi < n_words; wi += blockDim.x) {
        const uint64_t W = cs + (wi << 4);
        const uint64_t lo_v = W > start ? W : start;
        const uint64_t hi_v = (W + 16 < end) ? W + 16 : end;
        if (lo_v >= hi_v) continue;
        uint64_t k = find(lo_v - out_addr);
        const uint64_t p0 = pos_of(k), p1 = pos_of(k + 1);
        const uint64_t wrel = W - out_addr;
        if (lo_v == W && hi_v == W + 16 && p0 <= wrel && wrel + 16 <= p1) {
          const uint4 v = load16_any(a.arena + src_of(k) + (wrel - p0));
          *reinterpret_cast<uint4*>((uintptr_t)W) = v;
          continue;
        }
        // the word straddles members or an end of the output
        uint32_t wv[4] = {0u, 0u, 0u, 0u};
        uint64_t kk = k, kp0 = p0, kp1 = p1, ksrc = src_of(k);
#pragma unroll
        for (int t = 0; t < 16; ++t) {
          const uint64_t addr = W + t;
          if (addr < lo_v || addr >= hi_v) continue;
          const uint64_t rel = addr - out_addr;
          while (rel >= kp1) {
            ++kk;
            kp0 = kp1;
            kp1 = pos_of(kk + 1);
            ksrc = src_of(kk);
          }
          const uint8_t byte = __ldg(a.arena + ksrc + (rel - kp0));
          wv[t >> 2] |= (uint32_t)byte << (8 * (t & 3));
        }
        if (lo_v == W && hi_v == W + 16) {
          *reinterpret_cast<uint4*>((uintptr_t)W) = make_uint4(wv[0], wv[1], wv[2], wv[3]);
        } else {
#pragma unroll
          for (int t = 0; t < 16; ++t) {
            const uint64_t addr = W + t;
            if (addr >= lo_v && addr < hi_v)
              *reinterpret_cast<uint8_t*>((uintptr_t)addr) = (uint8_t)(wv[t >> 2] >> (8 * (t & 3)));
          }
        }
      }
      __syncthreads();
    }
  }
  if (threadIdx.x == 0) {
    __threadfence();
    if (atomicAdd(&ds->exit_ctr[TS_ASM_COPY], 1u) == gridDim.x - 1) {
      if (!failed && a.cursor) *a.cursor = base + S;
      if (a.out_bytes) *a.out_bytes = S;
      ds->as_err = 0u;
      ds->exit_ctr[TS_ASM_COPY] = 0u;
      __threadfence();
    }
  }
}

void launch_assemble(const LaunchCfg& L, const AssembleArgs& a) {
  RO_LAUNCH(L, K_APARENTS, (asm_parents_kernel<<<L.grid_aparents, AP_THREADS, 0, L.stream>>>(a)));
  RO_LAUNCH(L, K_AMEMBERS, (asm_members_kernel<<<L.grid_amembers, AM_THREADS, 0, L.stream>>>(a)));
  RO_LAUNCH(L, K_ACOPY, (asm_copy_kernel<<<L.grid_acopy, AC_THREADS, 0, L.stream>>>(a)));
}

const void* kernel_ptr_assemble(int which) {
  if (which == K_APARENTS) return (const void*)asm_parents_kernel;
  if (which == K_AMEMBERS) return (const void*)asm_members_kernel;
  return (const void*)asm_copy_kernel;
}

}  // namespace ro
