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
constexpr int CF_THREADS = 256, CF_WORDS = 4;                 // bitmap words per tile: 1024
constexpr int AP_THREADS = 256, AP_ITEMS = 4;                 // listed parents per tile: 1024
constexpr int AM_THREADS = 256, AM_ITEMS = 8;                 // members per tile: 2048
constexpr uint32_t AM_TILE = AM_THREADS * AM_ITEMS;
constexpr uint32_t AM_SMEM_CAP = 4096;                        // listed parents staged per tile
constexpr int AC_THREADS = 256;
constexpr uint64_t AC_CHUNK = 16384;                          // output bytes per copy chunk
constexpr uint32_t AC_BUF = 26624;                            // staged source bytes per chunk
constexpr uint32_t AC_PIECES = 640;                           // member pieces staged per chunk

// kernel entry points for occupancy queries and per-kernel timing
enum KernelId { K_EXPAND_SCAN, K_FILL, K_RB_COUNT, K_RB_SCATTER, K_COMMIT, K_CFINISH, K_APARENTS,
                K_AMEMBERS, K_ACOPY, K_COUNT };

// Launch counter and optional CUDA-event timing of selected kernels, on the
// stream they are launched on (see ro_ctx_profile in the C ABI).
struct Profiler;
void prof_begin(Profiler* p, cudaStream_t s, int kid);
void prof_end(Profiler* p, cudaStream_t s, int kid);

struct LaunchCfg {
  cudaStream_t stream;
  Profiler* prof;
  int grid_expand_scan, grid_fill, grid_rb, grid_commit, grid_cfinish, grid_aparents,
      grid_amembers, grid_acopy;
};

// launch one kernel between the profiler's marks
#define RO_LAUNCH(L, kid, ...)              \
  do {                                      \
    prof_begin((L).prof, (L).stream, kid);  \
    __VA_ARGS__;                            \
    prof_end((L).prof, (L).stream, kid);    \
  } while (0)

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
  uint32_t* phase;
  Rec* rec;
};
void launch_expand_fill(const LaunchCfg& L, const ExpandFillArgs& a);

// ---- ro_batch_ready ---------------------------------------------------------------
struct ReadyArgs {
  const uint32_t* cand;       // NULL: all children in id order
  uint64_t n_cand;
  uint64_t N;
  uint32_t* phase;
  const Rec* rec;             // read for the Call when the expansion has several
  int check_call;
  uint32_t call, batch_size;
  int flush;
  uint64_t cap;
  uint32_t* queue;            // this (expansion, Call) queue storage
  unsigned long long* qstate; // [head, tail]
  uint32_t* batched;
  uint64_t* n_batched_out;    // optional device output
  DevScalars* ds;
  TileStatus<unsigned long long> ts;
};
void launch_ready(const LaunchCfg& L, const ReadyArgs& a);

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
  uint32_t* phase;
  Rec* rec;
  unsigned long long* pw;
  uint32_t* bitmap;
  uint8_t* code;              // user's or internal
  uint32_t* done_user;        // optional
  uint32_t* done_int;
  uint64_t* n_done_out;       // optional device output
  // assembly plan of the completed parents (consumed by ro_assemble(NULL))
  const uint64_t* offsets;
  uint8_t* plan_status;       // P
  uint32_t* plan_mb;          // P+1 member bases
  uint32_t* plan_mtfp;        // member tile -> containing listed parent
  uint64_t plan_mtfp_cap;
  DevScalars* ds;
  TileStatus<Pair64> ts;
};
void launch_commit(const LaunchCfg& L, const CommitArgs& a);

// ---- ro_assemble ---------------------------------------------------------------------
struct AssembleArgs {
  const uint32_t* list;       // user's list or the latest commit's
  uint64_t n_host;            // list length, or capacity of the outputs
  const uint64_t* d_n;        // device list length (optional, user list only)
  int list_is_commit;         // plan of the latest commit (counts in ds->cm_n_done / cm_M)
  const uint8_t* plan_status; // that plan's statuses (copied to status), or NULL
  uint64_t P, N;
  const uint64_t* offsets;
  const unsigned long long* pw;
  const Rec* rec;
  const uint8_t* arena;
  uint64_t arena_bytes;
  uint8_t* status;
  uint64_t* out_off;
  uint32_t* out_len;          // optional
  uint8_t* out;
  uint64_t out_cap;
  uint64_t* cursor;           // optional (device)
  uint64_t* out_bytes;        // optional (device)
  // member bases / member-tile table: scratch (user list) or the commit's plan
  uint32_t* mb;               // member base per listed parent (n+1)
  uint32_t* mtfp;             // member tile -> containing listed parent
  uint64_t mtfp_cap;
  uint64_t* cpos;             // nonzero member output positions (relative to out)
  uint64_t* csrc;             // nonzero member arena offsets
  uint64_t member_cap;        // capacity of cpos/csrc
  uint32_t* ctfp;             // copy chunk -> first member
  uint64_t ctfp_cap;
  DevScalars* ds;
  TileStatus<unsigned long long> ts_parents;
  TileStatus<Pair64> ts_members;
};
void launch_assemble(const LaunchCfg& L, const AssembleArgs& a);


}  // namespace ro
