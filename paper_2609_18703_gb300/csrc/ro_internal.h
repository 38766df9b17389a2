// ro_internal.h — host-side declarations shared by the API and kernel files.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "ro_common.cuh"

namespace ro {

// Work sizes (elements per tile) of the scan kernels.
constexpr int EXP_THREADS = 256, EXP_ITEMS = 16;             // parents per scan tile: 4096
constexpr uint32_t FILL_TILE = 4096;                          // children per fill tile
constexpr int FILL_THREADS = 256;
constexpr uint32_t FILL_SMEM_CAP = FILL_TILE + 256;           // offsets staged per fill tile
constexpr int RB_THREADS = 256, RB_ITEMS = 8;                 // candidates per tile: 2048
constexpr int CM_THREADS = 256;
// commit_plan: a tile of CP_WORDS bitmap words (32 parents each, one word
// per thread; CP_WORDS <= CP_THREADS); at most CP_CAP completed parents staged in shared memory at a
// time, members in rounds of CP_ROUND.  At CP_MAXREG registers and ~27 KB of
// shared memory a CTA fits beside two asm_copy CTAs on one SM.
#ifndef RO_CP_WORDS
#define RO_CP_WORDS 256
#endif
constexpr int CP_THREADS = 256;
constexpr uint32_t CP_WORDS = RO_CP_WORDS;
static_assert(CP_WORDS <= (uint32_t)CP_THREADS, "one bitmap word per thread at most");
constexpr uint32_t CP_CAP = 2048;
constexpr int CP_ITEMS = 4;
constexpr uint32_t CP_ROUND = CP_THREADS * CP_ITEMS;
#define CP_MAXREG 56
constexpr int MB_ITEMS = 8;                                   // members per lane per step
constexpr int AP_THREADS = 256, AP_ITEMS = 4;                 // listed parents per tile: 1024
// members per tile: 1024.  At 56 registers and 17 KB of shared memory a CTA
// fits beside two asm_copy CTAs on one SM (2 x 320 x 80 + 256 x 56 = 65,536
// registers), so the next waves' planning runs while a copy is in flight.
constexpr int AM_THREADS = 256, AM_ITEMS = 4;
constexpr uint32_t AM_TILE = AM_THREADS * AM_ITEMS;
constexpr uint32_t AM_SMEM_CAP = 2048;                        // listed parents staged per tile
constexpr int AC_THREADS = 320;                               // 2 producer + 8 consumer warps
constexpr int AC_PRODUCERS = 2, AC_CONSUMERS = AC_THREADS / 32 - AC_PRODUCERS;
constexpr int AC_STAGES = 3;                                  // chunks staged per CTA
constexpr uint64_t AC_CHUNK = 16384;                          // output bytes per copy chunk (relative)
// A chunk is staged when it has at most AC_PIECES member pieces whose
// 16-byte-aligned source blocks fit AC_BUF bytes (each piece adds < 32 bytes
// of alignment to its payload); other chunks are copied directly.  Packed
// records of 32 bytes or more start on 16-byte boundaries and fit.
constexpr uint32_t AC_PIECES = 1024;
constexpr uint32_t AC_BUF = 24576;
constexpr uint32_t AC_SMALL = 64;   // pieces of at most this many staged bytes: cp.async, not a bulk copy
// copies of at most this many chunks take the direct path (RO_COPY_SMALL_CHUNKS
// in the environment at context creation overrides it; 0 stages every copy)
constexpr uint64_t AC_SMALL_CHUNKS = 256;

// kernel entry points for occupancy queries and per-kernel timing
enum KernelId { K_EXPAND_SCAN, K_FILL, K_RB_COUNT, K_RB_SCATTER, K_COMMIT, K_CPLAN, K_APARENTS,
                K_AMEMBERS, K_ACOPY, K_RT_CLAIM, K_RT_SCATTER, K_PB_KEYS, K_PB_HIST,
                K_PB_ROWSCAN, K_PB_SORT, K_PB_BOUNDS, K_PB_HEADS, K_PB_MARK, K_PB_SCAN, K_PB_EMIT,
                K_CFIX, K_RB_FUSED, K_COUNT,
                K_RB_FUSED_CALLS = 100 };   // occupancy query only (profiled as K_RB_FUSED)


// Launch counter and optional CUDA-event timing of selected kernels, on the
// stream they are launched on (see ro_ctx_profile in the C ABI).
struct Profiler;
void prof_begin(Profiler* p, cudaStream_t s, int kid);
void prof_end(Profiler* p, cudaStream_t s, int kid);

struct LaunchCfg {
  cudaStream_t stream;
  Profiler* prof;
  int grid_expand_scan, grid_fill, grid_rb, grid_commit, grid_cplan, grid_aparents,
      grid_amembers, grid_acopy, grid_retry, grid_pb, grid_pb_sort;
  // CTAs of the one-pass admission (one Call; several) the device holds at
  // once (0: no cooperative launch)
  int grid_rb_coop, grid_rb_coop_calls;
};

// Launch one kernel between the profiler's marks, with programmatic
// dependent launch: the kernel may be scheduled while its predecessor on the
// stream drains, and waits (griddepcontrol.wait, first statement of every
// kernel here) until the predecessor has finished and its writes are visible.
template <typename Arg>
inline void launch_k(const LaunchCfg& L, int kid, void (*kern)(Arg), int grid, int block,
                     size_t smem, const Arg& a) {
  prof_begin(L.prof, L.stream, kid);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3((unsigned)block);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = L.stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaLaunchKernelEx(&cfg, kern, a);
  prof_end(L.prof, L.stream, kid);
}

// The same for a kernel whose CTAs wait for one another (grid barriers): a
// cooperative launch, so that every CTA of the grid is resident at once (the
// grid must not exceed what the device holds; see LaunchCfg::grid_rb_coop),
// with programmatic dependent launch as above.
template <typename Arg>
inline void launch_coop(const LaunchCfg& L, int kid, void (*kern)(Arg), int grid, int block, const Arg& a) {
  prof_begin(L.prof, L.stream, kid);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3((unsigned)block);
  cfg.stream = L.stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  cudaLaunchKernelEx(&cfg, kern, a);
  prof_end(L.prof, L.stream, kid);
}

// ---- self-test of the bounded waits ---------------------------------------------------
struct SelftestArgs {
  uint32_t kind;              // 0: look-back on an unpublished tile; 1: grid barrier missing an arrival
  TileStatus<unsigned long long> ts;   // two tiles, flags zero
  unsigned long long epoch;   // an epoch no flag holds
  ReadyScalars* rs;           // barrier scratch, zeroed
  uint32_t* err;
};
void launch_selftest(cudaStream_t s, const SelftestArgs& a);

// ---- ro_expand ----------------------------------------------------------------
struct ExpandScanArgs {
  const uint32_t* counts;
  uint64_t P;
  uint64_t* offsets_user;
  uint64_t* offsets;          // internal copy
  unsigned long long* pw;     // per-parent remaining | bad
  uint32_t* empty_out;        // optional
  uint32_t* tfp;              // fill tile -> parent of its first child
  uint64_t tfp_cap;           // entries available in tfp
  DevScalars* ds;
  TileStatus<Pair64> ts;
};
void launch_expand_scan(const LaunchCfg& L, const ExpandScanArgs& a);

struct ExpandFillArgs {
  const uint64_t* offsets;
  uint64_t P, N;
  const uint32_t* tfp;
  const uint8_t* parent_call;  // optional
  uint32_t* child_parent;
  uint32_t* child_ordinal;
  Slot* slot;
  uint32_t* par;
};
void launch_expand_fill(const LaunchCfg& L, const ExpandFillArgs& a);

// ---- ro_batch_ready ---------------------------------------------------------------
struct ReadyArgs {
  const uint32_t* cand;       // NULL: all children in id order
  uint64_t n_cand;
  uint64_t N;
  Slot* slot;                 // phase word; the Call (w) when the expansion has several
  int check_call;
  int calls_concurrent;       // other Calls' admissions may run at the same time
  uint32_t call, batch_size;
  int flush;
  uint64_t cap;
  uint32_t* queue;            // this (expansion, Call) queue storage
  unsigned long long* qstate; // [head, tail, recovery length]
  const uint32_t* rq;         // this (expansion, Call) recovery queue storage
  uint32_t* batched;
  uint64_t* n_batched_out;    // optional device output
  int parent_bound;           // admit only: the window is reserved by launch_parent
  DevScalars* ds;
  ReadyScalars* rs;           // this Call's
  TileStatus<unsigned long long> ts;   // this Call's
};
void launch_ready(const LaunchCfg& L, const ReadyArgs& a);
// the admissions of up to RB_CALLS_MAX Calls from one candidate list, one
// cooperative launch (the caller checks that the grid fits: LaunchCfg::grid_rb_coop_calls)
constexpr uint32_t RB_CALLS_MAX = 8;
struct MultiReadyArgs {
  ReadyArgs a[RB_CALLS_MAX];
  uint32_t n;
};
void launch_ready_calls(const LaunchCfg& L, const MultiReadyArgs& m);
// ---- ro_batch_ready_parent ---------------------------------------------------------
constexpr int PB_THREADS = 256, PB_ITEMS = 8;                 // queue entries per tile: 2048
constexpr uint32_t PB_TILE = PB_THREADS * PB_ITEMS;
constexpr int PB_DIGITS = 256;                                // radix of the sort by parent
struct ParentArgs {
  uint64_t N, P;
  uint32_t B;
  int flush;
  int passes;                 // 8-bit digit passes covering the largest parent id
  int pass;                   // the sort pass of this launch
  const uint32_t* par;
  Slot* slot;
  uint32_t* queue;
  unsigned long long* qstate;
  uint32_t* batched;
  uint64_t cap;
  uint64_t* batch_off;        // optional
  uint64_t off_cap;
  uint64_t* n_batched_out;    // optional
  uint64_t* n_batches_out;    // optional
  // scratch; per window entry (at most N of them) unless noted
  uint32_t* key[2];           // parent of the entry, sorted by passes
  uint32_t* val[2];           // window position of the entry, permuted alike
  uint32_t* child;            // the window's children
  uint32_t* hist;             // PB_DIGITS x tiles, digit-major
  uint32_t* dtot;             // PB_DIGITS digit totals
  uint32_t* first;            // per parent: sorted position of its first entry
  uint32_t* endp;             // per parent: one past its last
  uint32_t* hsz;              // by queue position: chunk size at a chunk's first entry, else 0
  uint8_t* left;              // by queue position: 1 if the entry stays queued (no flush)
  uint32_t* hoff;             // by queue position of a taken chunk's first entry: output offset
  uint32_t* rem;              // entries left in the queue, in order
  DevScalars* ds;
  TileStatus<Pair64> ts;
};
void launch_parent(const LaunchCfg& L, const ParentArgs& a);

// ---- ro_retry ----------------------------------------------------------------------
constexpr int RT_THREADS = 256, RT_ITEMS = 8;                 // retry entries per tile: 2048
struct RetryArgs {
  const uint32_t* children;
  uint64_t n;
  uint64_t N;
  Slot* slot;                 // len of an IN-FLIGHT Grain holds the claim (~index) meanwhile
  int check_call;
  uint32_t call;
  uint32_t* rq;               // recovery queue storage
  unsigned long long* qstate; // [head, tail, recovery length]
  DevScalars* ds;
  TileStatus<unsigned long long> ts;
};
void launch_retry(const LaunchCfg& L, const RetryArgs& a);

// ---- lists and plans -------------------------------------------------------------------
// A list of parents to assemble with its member bases: produced by
// commit_plan (the parents a commit completed) or by asm_parents (a
// caller's list), consumed by asm_members.
struct ListBufs {
  const uint32_t* parents;    // listed parent ids
  uint8_t* status;            // outcome per listed parent
  uint32_t* mb;               // member base per listed parent (+ total at [n])
  uint32_t* coff;             // first child of each listed parent
  uint32_t* mtfp;             // member tile -> listed parent holding its first member
  uint64_t mtfp_cap;
  ListHdr* hdr;
};
// The assembly plan of a list: everything the copy needs, with positions
// relative to the start of that call's output.  Produced by asm_members, or
// by commit_plan for the commit's own list; consumed by asm_copy.
struct PlanBufs {
  uint64_t* off;              // relative output offset per listed parent (+ total at [n])
  uint64_t* cpos;             // relative output position of each contributing member
  uint64_t* csrc;             // arena offset of each contributing member
  uint64_t member_cap;        // capacity of cpos / csrc
  uint32_t* ctfp;             // relative 16 KB chunk -> member holding its first byte
  uint64_t ctfp_cap;
  PlanHdr* hdr;
};

// ---- ro_gather_commit ----------------------------------------------------------------
struct CommitArgs {
  uint64_t n_host;
  const uint64_t* d_n;        // optional device count
  const uint32_t* child;
  const uint8_t* state;
  const uint32_t* len;
  const uint64_t* off;
  const uint32_t* gen;        // optional
  uint64_t arena_bytes;
  uint64_t N, P;
  Slot* slot;
  const uint32_t* par;
  unsigned long long* pw;
  uint32_t* bitmap;           // parents this call completed
  int heavy;                  // heavy parents hold a quarter of the children: count them per CTA first
  const uint32_t* tfp;        // fill tile -> parent of its first child (expand_fill's table)
  uint64_t n_fill_tiles;      // tiles of FILL_TILE children written in tfp
  unsigned long long* gb;     // per parent: (seq << 32) | ~r for the lowest accepted
                              // GroupFailure report r of commit seq; older seq: none
  uint32_t seq;               // this commit's sequence number in the context (from 1)
  uint8_t* code;              // user's or internal
  uint32_t* done_user;        // optional
  uint32_t* done_int;         // the list (a ring slot)
  uint64_t* n_done_out;       // optional device output
  const uint64_t* offsets;
  ListBufs list;              // written: the completed parents with member bases
  PlanBufs plan;              // written: the copy plan of that list
  int pslot;                  // commit_plan's scan slot (commit sequence modulo FIN_STREAMS)
  DevScalars* ds;
  TileStatus<Quad64> tsq;     // commit_plan's look-back
};
// the scatter (then the fix-up of repeated reports and GroupFailure
// barriers) and the completion list with its copy plan, which may run on
// different streams
void launch_commit_scatter(const LaunchCfg& L, const CommitArgs& a);
void launch_commit_plan(const LaunchCfg& L, const CommitArgs& a);

// ---- ro_assemble ---------------------------------------------------------------------
struct AssembleArgs {
  const uint32_t* user_list;  // explicit list (asm_parents), or NULL: the commit's list
  uint64_t n_host;            // list length, or capacity of the per-parent outputs
  const uint64_t* d_n;        // device list length (optional, explicit list only)
  uint64_t P, N;
  const uint64_t* offsets;
  const unsigned long long* pw;
  const Slot* slot;
  const uint8_t* arena;
  uint64_t arena_bytes;
  int arena_host;             // the arena is pinned host memory: no bulk (TMA) copies from it
  uint64_t small_chunks;      // copies of at most this many chunks go direct (no staging)
  uint8_t* status;
  uint64_t* out_off;
  uint32_t* out_len;          // optional
  uint8_t* out;
  uint64_t out_cap;
  uint64_t* cursor;           // optional (device)
  uint64_t* out_bytes;        // optional (device)
  // list structure (optional; ro_assemble_list): per listed parent its first
  // entry, per entry (member of a Present parent) outcome, offset, length
  uint64_t* elem_base;
  uint8_t* elem_state;
  uint64_t* elem_off;
  uint32_t* elem_len;
  uint64_t elem_cap;
  uint64_t* n_elems_out;      // optional (device)
  ListBufs list;
  PlanBufs plan;
  DevScalars* ds;
  TileStatus<unsigned long long> ts_parents;
  TileStatus<Pair64> ts_members;
};
// the planning kernels (explicit lists: asm_parents then asm_members) and
// the copy, each on its own stream
void launch_assemble_plan(const LaunchCfg& L, const AssembleArgs& a);
void launch_assemble_copy(const LaunchCfg& L, const AssembleArgs& a);
// F.filter on a report batch (context-free)
void launch_filter(cudaStream_t s, uint8_t* state, const uint8_t* keep, uint64_t n, int grid);



}  // namespace ro
