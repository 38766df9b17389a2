// ro_api.cu — host side of the C ABI declared in include/rayorch_gpu.h:
// argument checks, ownership of the per-expansion device state, scratch,
// kernel launches on the context's streams, and the mapping of
// device-recorded conditions to statuses.
//
// Streams.  Expansion, admission and commit run on the context's stream.
// Assembly planning (asm_parents, asm_members) runs on the plan stream and
// the copy on the copy stream; both default to the context's stream.  With
// separate streams the work of consecutive waves overlaps: the lists of
// completed parents and the assembly plans live in rings of slots per
// expansion, handed from stream to stream with events.
#include <algorithm>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <string>
#include <vector>

#include "../../include/rayorch_gpu.h"
#include "ro_internal.h"

namespace ro {
cudaError_t prepare_assemble_kernels();
size_t asm_copy_smem();
const void* kernel_ptr_expand(int which);
const void* kernel_ptr_ready(int which);
const void* kernel_ptr_commit(int which);
const void* kernel_ptr_complete();
const void* kernel_ptr_assemble(int which);
const void* kernel_ptr_retry(int which);
const void* kernel_ptr_parent(int which);
}  // namespace ro

using namespace ro;

namespace {

constexpr int MAX_EXPANSIONS = 64;
constexpr int N_TS = N_TILE_SLOTS;    // tile-status slots (TS_* in ro_common.cuh)
constexpr int RING = FIN_STREAMS + 1 > 3 ? FIN_STREAMS + 1 : 3;   // list / plan slots per expansion
// Completion bitmaps per expansion, taken in turn by its commits.  A commit
// may reuse a slot once the plan that read it (BM_SLOTS commits earlier) is
// done; the context's stream waits for that only every BM_WAIT commits (for
// all plans at least BM_WAIT + 1 commits old), so a scatter seldom depends
// on anything but the previous kernel on its stream and launches early.
#ifndef RO_BM_SLOTS
#define RO_BM_SLOTS 32
#endif
constexpr int BM_SLOTS = RO_BM_SLOTS;
constexpr int BM_WAIT = BM_SLOTS / 2;

struct DevBuf {
  void* p = nullptr;
  size_t cap = 0;
};

// An event with the stream capture it was recorded under (0: none).
struct Ev {
  cudaEvent_t e = nullptr;
  unsigned long long cap_id = 0;
  bool recorded = false;
};

struct QueueBufs {
  DevBuf q, rq, state;  // Ready Queue, recovery queue, [head, tail, recovery length]
  bool ready = false;   // state zeroed for the current expansion
};

// A list of completed parents with its copy plan (written by a commit's
// commit_plan; read by the copy, or by planning for an explicit assembly).
struct ListSlot {
  DevBuf done, status, mb, coff, mtfp, hdr;
  DevBuf poff, pcpos, pcsrc, pctfp, phdr;   // the copy plan
  uint64_t pctfp_cap = 0;
  Ev freed;     // the assembly that read it is done
  Ev planned;   // the commit_plan that wrote it is done (the next writer may run on the other stream)
};
// An assembly plan (written by planning, read by the copy).
struct PlanSlot {
  DevBuf off, cpos, csrc, ctfp, hdr;
  uint64_t ctfp_cap = 0;
  Ev ready, freed;
};

// Device buffers of one expansion slot, kept across ro_ctx_reset and reused.
struct ExpSlot {
  DevBuf offsets, pw, slot, par, bitmap, tfp, gb;   // bitmap: BM_SLOTS slots
  Ev bm_free[BM_SLOTS];   // the plan that read a bitmap slot is done
  int bm_stream[BM_SLOTS] = {};   // the completion stream that plan ran on
  ListSlot lists[RING];
  PlanSlot plans[RING];
  std::vector<QueueBufs> queues;
};

struct Expansion {
  int32_t parent_xid = -1;
  uint64_t P = 0, N = 0;
  uint64_t commits = 0, assembles = 0;
  int last_list = -1;   // list slot written by the latest commit
  bool heavy = false;   // parents of at least HEAVY_CHILDREN children hold >= N/4 children
};

struct TsBuf {
  DevBuf flag, agg, inc;
};

}  // namespace

namespace ro {
// Launch counts always; CUDA-event pairs around the kernels selected by mask.
struct Profiler {
  uint32_t mask = 0;
  std::vector<cudaEvent_t> pool;
  size_t used = 0;
  std::vector<std::pair<int, size_t>> marks;   // (kernel, index of its start event)
  uint64_t launches[K_COUNT] = {};
  uint64_t timed[K_COUNT] = {};
  double ms[K_COUNT] = {};
  int pending = -1;
};

void prof_begin(Profiler* p, cudaStream_t s, int kid) {
  if (!p) return;
  p->launches[kid] += 1;
  p->pending = -1;
  if (!(p->mask & (1u << kid))) return;
  if (p->used + 2 > p->pool.size()) {
    const size_t add = std::max<size_t>(p->pool.size(), 256);
    for (size_t i = 0; i < add; ++i) {
      cudaEvent_t e;
      if (cudaEventCreate(&e) != cudaSuccess) {
        cudaGetLastError();
        return;
      }
      p->pool.push_back(e);
    }
  }
  cudaEventRecord(p->pool[p->used], s);
  p->pending = (int)p->used;
  p->used += 2;
}

void prof_end(Profiler* p, cudaStream_t s, int kid) {
  if (!p || p->pending < 0) return;
  cudaEventRecord(p->pool[p->pending + 1], s);
  p->marks.emplace_back(kid, (size_t)p->pending);
  p->pending = -1;
}
}  // namespace ro

struct ro_ctx {
  int device = 0;
  cudaStream_t stream = nullptr;        // expansion, admission, commit
  cudaStream_t plan_stream = nullptr;   // assembly planning
  cudaStream_t copy_stream = nullptr;   // assembly copies
  // Completion lists and their plans (commit_plan): with separate streams,
  // consecutive commits take FIN_STREAMS streams in turn, so the plans of
  // consecutive commits run at the same time.
  cudaStream_t fin_stream[FIN_STREAMS] = {};
  cudaStream_t own_fin[FIN_STREAMS] = {};   // created for fin_stream, destroyed with the context
  int last_fin = 0;                     // the stream of the latest commit's plan
  uint32_t n_calls = 1;
  uint32_t commit_seq = 0;              // commits issued on this context
  uint64_t copy_small_chunks = AC_SMALL_CHUNKS;   // copies this small go direct
  int num_sms = 0;
  LaunchCfg L{}, Lp{}, Lc{}, Lf[FIN_STREAMS]{};
  DevScalars* ds = nullptr;
  DevScalars* hs = nullptr;   // pinned mirror
  ReadyScalars* rs = nullptr;   // per Call, device
  ReadyScalars* hrs = nullptr;  // per Call, pinned mirror
  // Streams of the Calls' admissions (ro_ctx_set_call_streams; the
  // context's stream when unset).  An admission on a Call's stream follows
  // the context's stream (call_fork); the context's stream waits for it
  // (call_join) before its next launch of its own.
  std::vector<cudaStream_t> call_stream;
  std::vector<Ev> call_fork, call_join;
  std::vector<char> call_pending;
  std::vector<TsBuf> ts_call;   // the admission scans' tile status, per Call
  std::vector<ExpSlot> slots;
  std::vector<Expansion> exps;
  TsBuf ts[N_TS];
  DevBuf code;
  DevBuf selftest;                      // ro_ctx_selftest_timeout scratch
  DevBuf x_mb, x_coff, x_mtfp, x_hdr;   // explicit-list assembly scratch
  // parent-bound reservation scratch (see ParentArgs)
  DevBuf pb_key[2], pb_val[2], pb_child, pb_hist, pb_dtot, pb_first, pb_endp, pb_hsz, pb_left,
      pb_hoff, pb_rem;
  Ev fork, x_planned, join_plan, join_copy, fin_fork[FIN_STREAMS], fin_join[FIN_STREAMS], fin_plan;
  // Caller memory written by the copies issued since the context's stream
  // last waited for the copy stream: a later call's planning (another
  // stream) may run while they do, so planning that writes any of it waits
  // for them (copy_done follows the latest copy).  Past MAX_SPANS ranges
  // every such planning waits.
  struct Span {
    uintptr_t lo, hi;
  };
  static constexpr size_t MAX_SPANS = 4096;
  std::vector<Span> copy_spans;
  bool copy_spans_full = false;
  Ev copy_done;
  Profiler prof;
  ro_status sticky = RO_OK;
  std::string err;
};

namespace {

struct DeviceGuard {
  int prev = -1;
  explicit DeviceGuard(int dev) {
    int cur = -1;
    if (cudaGetDevice(&cur) == cudaSuccess && cur != dev) {
      prev = cur;
      cudaSetDevice(dev);
    }
  }
  ~DeviceGuard() {
    if (prev >= 0) cudaSetDevice(prev);
  }
};

ro_status fail(ro_ctx* c, ro_status st, const char* fmt, ...) __attribute__((format(printf, 3, 4)));
ro_status fail(ro_ctx* c, ro_status st, const char* fmt, ...) {
  if (c) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    c->err = buf;
  }
  return st;
}

ro_status cuda_fail(ro_ctx* c, cudaError_t e, const char* what) {
  c->sticky = RO_E_CUDA;
  return fail(c, RO_E_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

#define RO_TRY(x)                 \
  do {                            \
    ro_status _s = (x);           \
    if (_s != RO_OK) return _s;   \
  } while (0)

unsigned long long capture_id(cudaStream_t s) {
  cudaStreamCaptureStatus st = cudaStreamCaptureStatusNone;
  unsigned long long id = 0;
  if (cudaStreamGetCaptureInfo(s, &st, &id) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return st == cudaStreamCaptureStatusActive ? id : 0;
}

void sync_all_streams(ro_ctx* c) {
  cudaStreamSynchronize(c->stream);
  if (c->plan_stream != c->stream) cudaStreamSynchronize(c->plan_stream);
  if (c->copy_stream != c->stream) cudaStreamSynchronize(c->copy_stream);
  for (cudaStream_t s : c->fin_stream)
    if (s != c->stream) cudaStreamSynchronize(s);
  for (cudaStream_t s : c->call_stream)
    if (s != c->stream) cudaStreamSynchronize(s);
}

// Grow-only device buffer, zeroed when (re)allocated.  Growth needs a
// synchronisation, so it is refused while the context's stream is captured.
ro_status ensure(ro_ctx* c, DevBuf& b, size_t bytes, const char* what) {
  if (bytes == 0) bytes = 16;
  if (b.cap >= bytes) return RO_OK;
  if (capture_id(c->stream))
    return fail(c, RO_E_STATE, "%s must grow during stream capture: run the call once uncaptured first", what);
  if (b.p) {
    sync_all_streams(c);   // the old buffer may be in use on any stream
    cudaFree(b.p);
    b.p = nullptr;
    b.cap = 0;
  }
  size_t want = bytes + bytes / 8;   // a little headroom for the next, larger call
  want = (want + 255) & ~(size_t)255;
  cudaError_t e = cudaMalloc(&b.p, want);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return fail(c, RO_E_OOM, "cannot allocate %zu bytes for %s", want, what);
  }
  b.cap = want;
  e = cudaMemsetAsync(b.p, 0, want, c->stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(c->stream);   // zero before any stream uses it
  if (e != cudaSuccess) return cuda_fail(c, e, "cudaMemsetAsync");
  return RO_OK;
}

ro_status ev_record(ro_ctx* c, Ev& ev, cudaStream_t s) {
  if (!ev.e) {
    cudaError_t e = cudaEventCreateWithFlags(&ev.e, cudaEventDisableTiming);
    if (e != cudaSuccess) return cuda_fail(c, e, "cudaEventCreate");
  }
  cudaError_t e = cudaEventRecord(ev.e, s);
  if (e != cudaSuccess) return cuda_fail(c, e, "cudaEventRecord");
  ev.cap_id = capture_id(s);
  ev.recorded = true;
  return RO_OK;
}

// Make s wait for ev.  An event recorded in the capture that is now active on
// the context's stream is waited on (pulling s into that capture if it is
// not in it yet); an event recorded outside any capture is waited on only by
// a stream that is not being captured; an event from a finished capture is
// skipped.  What is skipped is ordered through the context's stream: a
// captured graph joins its streams back into it, and the caller joins the
// streams before it starts a capture.
ro_status ev_wait(ro_ctx* c, const Ev& ev, cudaStream_t s) {
  if (!ev.recorded) return RO_OK;
  const unsigned long long cs = capture_id(s);
  if (ev.cap_id == 0) {
    if (cs != 0) return RO_OK;
  } else {
    const unsigned long long active = capture_id(c->stream);
    if (ev.cap_id != active || (cs != 0 && cs != active)) return RO_OK;
  }
  cudaError_t e = cudaStreamWaitEvent(s, ev.e, 0);
  if (e != cudaSuccess) return cuda_fail(c, e, "cudaStreamWaitEvent");
  return RO_OK;
}

// from -> to: `to` waits for everything enqueued on `from` so far
ro_status order(ro_ctx* c, Ev& ev, cudaStream_t from, cudaStream_t to) {
  if (from == to) return RO_OK;
  RO_TRY(ev_record(c, ev, from));
  return ev_wait(c, ev, to);
}

// The context's stream waits for the plan and copy streams.
// The context's stream waits for the admissions still pending on the Calls'
// streams; every launch of its own (and every fork from it) comes after.
ro_status settle_calls(ro_ctx* c) {
  for (size_t k = 0; k < c->call_pending.size(); ++k) {
    if (!c->call_pending[k]) continue;
    RO_TRY(order(c, c->call_join[k], c->call_stream[k], c->stream));
    c->call_pending[k] = 0;
  }
  return RO_OK;
}

ro_status join(ro_ctx* c) {
  RO_TRY(settle_calls(c));
  for (int k = 0; k < FIN_STREAMS; ++k) RO_TRY(order(c, c->fin_join[k], c->fin_stream[k], c->stream));
  RO_TRY(order(c, c->join_plan, c->plan_stream, c->stream));
  if (c->copy_stream != c->plan_stream) RO_TRY(order(c, c->join_copy, c->copy_stream, c->stream));
  // planning forks from the context's stream: it now follows every copy
  c->copy_spans.clear();
  c->copy_spans_full = false;
  return RO_OK;
}

// Tile-status arrays of one scan slot (flags start zeroed: epoch 0, nothing
// published; kernels keep their epochs on the device).
template <class T>
ro_status tile_status_buf(ro_ctx* c, TsBuf& t, size_t tiles, TileStatus<T>* out) {
  tiles = std::max<size_t>(tiles, 1);
  const size_t el = std::max(sizeof(T), sizeof(Pair64));
  RO_TRY(ensure(c, t.flag, tiles * sizeof(unsigned long long), "scan flags"));
  RO_TRY(ensure(c, t.agg, tiles * el, "scan aggregates"));
  RO_TRY(ensure(c, t.inc, tiles * el, "scan prefixes"));
  out->flag = (unsigned long long*)t.flag.p;
  out->agg = (T*)t.agg.p;
  out->inc = (T*)t.inc.p;
  return RO_OK;
}
template <class T>
ro_status tile_status(ro_ctx* c, int slot, size_t tiles, TileStatus<T>* out) {
  return tile_status_buf(c, c->ts[slot], tiles, out);
}

ro_status check_launch(ro_ctx* c, const char* what) {
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(c, e, what);
  return RO_OK;
}

// Wait for every stream, mirror the device scalars and turn recorded
// conditions into a status (clearing them).
ro_status sync_and_check(ro_ctx* c) {
  RO_TRY(join(c));
  cudaError_t e = cudaMemcpyAsync(c->hs, c->ds, sizeof(DevScalars), cudaMemcpyDeviceToHost, c->stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(c->stream);
  if (e != cudaSuccess) return cuda_fail(c, e, "synchronise");
  const uint32_t err = c->hs->err;
  if (!err) return RO_OK;
  cudaMemsetAsync(&c->ds->err, 0, sizeof(uint32_t), c->stream);
  if (err & ERR_TIMEOUT)
    return fail(c, RO_E_TIMEOUT, (err & ERR_DRAIN)
                                     ? "a device-side wait timed out (a copy CTA exited with bulk "
                                       "copies still in flight)"
                                     : "a device-side wait timed out");
  if (err & ERR_OVERFLOW) return fail(c, RO_E_OVERFLOW, "an assembled parent exceeds 2^32-1 bytes");
  if (err & ERR_CAPACITY) return fail(c, RO_E_CAPACITY, "an output buffer is too small");
  return fail(c, RO_E_INVAL, "a device count or arena offset exceeded its bound");
}

ro_status enter(ro_ctx* c) {
  if (!c) return RO_E_INVAL;
  if (c->sticky != RO_OK) return c->sticky;
  c->err.clear();
  return RO_OK;
}

Expansion* get_exp(ro_ctx* c, int32_t xid) {
  if (xid < 0 || xid >= (int32_t)c->exps.size()) return nullptr;
  return &c->exps[xid];
}

int grid_for(const void* k, int threads, int sms, int cap_per_sm, size_t dyn_smem = 0) {
  int per = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per, k, threads, dyn_smem) != cudaSuccess || per < 1) {
    cudaGetLastError();
    per = 1;
  }
  per = std::min(per, cap_per_sm);
  return per * sms;
}

void free_buf(DevBuf& b) {
  if (b.p) cudaFree(b.p);
  b.p = nullptr;
  b.cap = 0;
}
void free_ev(Ev& e) {
  if (e.e) cudaEventDestroy(e.e);
  e = Ev{};
}

ListBufs list_bufs(ListSlot& s, uint64_t mtfp_cap) {
  ListBufs l;
  l.parents = (const uint32_t*)s.done.p;
  l.status = (uint8_t*)s.status.p;
  l.mb = (uint32_t*)s.mb.p;
  l.coff = (uint32_t*)s.coff.p;
  l.mtfp = (uint32_t*)s.mtfp.p;
  l.mtfp_cap = mtfp_cap;
  l.hdr = (ListHdr*)s.hdr.p;
  return l;
}

PlanBufs list_plan_bufs(ListSlot& s, uint64_t member_cap) {
  PlanBufs p;
  p.off = (uint64_t*)s.poff.p;
  p.cpos = (uint64_t*)s.pcpos.p;
  p.csrc = (uint64_t*)s.pcsrc.p;
  p.member_cap = member_cap;
  p.ctfp = (uint32_t*)s.pctfp.p;
  p.ctfp_cap = s.pctfp_cap;
  p.hdr = (PlanHdr*)s.phdr.p;
  return p;
}

PlanBufs plan_bufs(PlanSlot& s, uint64_t member_cap) {
  PlanBufs p;
  p.off = (uint64_t*)s.off.p;
  p.cpos = (uint64_t*)s.cpos.p;
  p.csrc = (uint64_t*)s.csrc.p;
  p.member_cap = member_cap;
  p.ctfp = (uint32_t*)s.ctfp.p;
  p.ctfp_cap = s.ctfp_cap;
  p.hdr = (PlanHdr*)s.hdr.p;
  return p;
}

// The device's view of a caller pointer: device memory as is; pinned host
// memory through its device mapping (*host = 1); pageable host memory is an
// error (the GPU may not reach it).
template <class T>
ro_status device_view(ro_ctx* c, T* p, T** out, int* host, const char* what) {
  cudaPointerAttributes at{};
  *host = 0;
  *out = p;
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return fail(c, RO_E_INVAL, "ro_assemble: %s pointer is not known to CUDA", what);
  }
  if (at.type == cudaMemoryTypeHost) {
    if (!at.devicePointer) return fail(c, RO_E_INVAL, "ro_assemble: %s host memory is not mapped", what);
    *out = (T*)at.devicePointer;
    *host = 1;
  } else if (at.type == cudaMemoryTypeUnregistered) {
    return fail(c, RO_E_INVAL, "ro_assemble: %s is pageable host memory (pin it)", what);
  }
  return RO_OK;
}

// The (expansion, Call) queues, empty at the expansion's first use.
ro_status queue_ready(ro_ctx* c, QueueBufs& Q, uint64_t N) {
  if (Q.ready) return RO_OK;
  RO_TRY(ensure(c, Q.q, N * sizeof(uint32_t), "ready queue"));
  RO_TRY(ensure(c, Q.rq, N * sizeof(uint32_t), "recovery queue"));
  RO_TRY(ensure(c, Q.state, 3 * sizeof(unsigned long long), "queue state"));
  cudaMemsetAsync(Q.state.p, 0, 3 * sizeof(unsigned long long), c->stream);
  Q.ready = true;
  return RO_OK;
}

void free_scalars(ro_ctx* c) {
  if (c->ds) cudaFree(c->ds);
  if (c->hs) cudaFreeHost(c->hs);
  if (c->rs) cudaFree(c->rs);
  if (c->hrs) cudaFreeHost(c->hrs);
  c->ds = nullptr;
  c->hs = nullptr;
  c->rs = nullptr;
  c->hrs = nullptr;
}

}  // namespace

extern "C" {

ro_status ro_ctx_create(ro_ctx** out, int32_t device, void* stream, uint32_t n_calls) {
  if (!out) return RO_E_INVAL;
  *out = nullptr;
  if (n_calls == 0 || n_calls > 256) return RO_E_INVAL;
  int ndev = 0;
  if (cudaGetDeviceCount(&ndev) != cudaSuccess || device < 0 || device >= ndev) {
    cudaGetLastError();
    return RO_E_CUDA;
  }
  DeviceGuard g(device);
  ro_ctx* c = new ro_ctx();
  c->device = device;
  c->stream = (cudaStream_t)stream;
  c->plan_stream = c->stream;
  c->copy_stream = c->stream;
  for (auto& f : c->fin_stream) f = c->stream;
  c->n_calls = n_calls;
  if (const char* e = std::getenv("RO_COPY_SMALL_CHUNKS")) c->copy_small_chunks = std::strtoull(e, nullptr, 10);
  cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, device);
  if (cudaMalloc(&c->ds, sizeof(DevScalars)) != cudaSuccess ||
      cudaMallocHost(&c->hs, sizeof(DevScalars)) != cudaSuccess ||
      cudaMalloc(&c->rs, n_calls * sizeof(ReadyScalars)) != cudaSuccess ||
      cudaMallocHost(&c->hrs, n_calls * sizeof(ReadyScalars)) != cudaSuccess) {
    cudaGetLastError();
    free_scalars(c);
    delete c;
    return RO_E_OOM;
  }
  cudaMemsetAsync(c->ds, 0, sizeof(DevScalars), c->stream);
  cudaMemsetAsync(c->rs, 0, n_calls * sizeof(ReadyScalars), c->stream);
  std::memset(c->hs, 0, sizeof(DevScalars));
  std::memset(c->hrs, 0, n_calls * sizeof(ReadyScalars));
  c->call_stream.assign(n_calls, c->stream);
  c->call_fork.resize(n_calls);
  c->call_join.resize(n_calls);
  c->call_pending.assign(n_calls, 0);
  c->ts_call.resize(n_calls);
  if (prepare_assemble_kernels() != cudaSuccess) {
    cudaGetLastError();
    free_scalars(c);
    delete c;
    return RO_E_CUDA;
  }
  const int s = c->num_sms;
  c->L.stream = c->stream;
  c->L.prof = &c->prof;
  c->L.grid_expand_scan = grid_for(kernel_ptr_expand(K_EXPAND_SCAN), EXP_THREADS, s, 4);
  c->L.grid_fill = grid_for(kernel_ptr_expand(K_FILL), FILL_THREADS, s, 8);
  c->L.grid_rb = grid_for(kernel_ptr_ready(K_RB_SCATTER), RB_THREADS, s, 8);
  {
    int coop = 0;
    cudaDeviceGetAttribute(&coop, cudaDevAttrCooperativeLaunch, device);
    c->L.grid_rb_coop = coop ? grid_for(kernel_ptr_ready(K_RB_FUSED), RB_THREADS, s, 64) : 0;
    c->L.grid_rb_coop_calls = coop ? grid_for(kernel_ptr_ready(K_RB_FUSED_CALLS), RB_THREADS, s, 64) : 0;
    // RO_ADMIT_TWO_PASS=1 in the environment at context creation keeps every
    // admission on the two-pass path
    if (const char* e = std::getenv("RO_ADMIT_TWO_PASS"))
      if (std::strtoul(e, nullptr, 10) != 0) c->L.grid_rb_coop = c->L.grid_rb_coop_calls = 0;
  }
  c->L.grid_commit = grid_for(kernel_ptr_commit(K_COMMIT), CM_THREADS, s, 8);
  c->L.grid_cplan = grid_for(kernel_ptr_complete(), CP_THREADS, s, 4);
  c->L.grid_aparents = grid_for(kernel_ptr_assemble(K_APARENTS), AP_THREADS, s, 4);
  // up to 4 planning CTAs per SM: large waves (100k-member parents) get the
  // parallelism; beside a running copy only one fits and the rest wait
  c->L.grid_amembers = grid_for(kernel_ptr_assemble(K_AMEMBERS), AM_THREADS, s, 4);
  c->L.grid_acopy = grid_for(kernel_ptr_assemble(K_ACOPY), AC_THREADS, s, 2, asm_copy_smem());
  c->L.grid_retry = grid_for(kernel_ptr_retry(K_RT_SCATTER), RT_THREADS, s, 4);
  c->L.grid_pb = grid_for(kernel_ptr_parent(K_PB_HEADS), PB_THREADS, s, 8);
  c->L.grid_pb_sort = grid_for(kernel_ptr_parent(K_PB_SORT), PB_THREADS, s, 8);
  c->Lp = c->L;
  c->Lc = c->L;
  for (auto& f : c->Lf) f = c->L;
  cudaError_t e = cudaStreamSynchronize(c->stream);
  if (e != cudaSuccess) {
    free_scalars(c);
    delete c;
    return RO_E_CUDA;
  }
  *out = c;
  return RO_OK;
}

ro_status ro_ctx_destroy(ro_ctx* c) {
  if (!c) return RO_E_INVAL;
  DeviceGuard g(c->device);
  sync_all_streams(c);
  for (auto& s : c->slots) {
    free_buf(s.offsets); free_buf(s.pw); free_buf(s.slot); free_buf(s.par); free_buf(s.bitmap);
    free_buf(s.tfp); free_buf(s.gb);
    for (auto& e : s.bm_free) free_ev(e);
    for (auto& l : s.lists) {
      free_buf(l.done); free_buf(l.status); free_buf(l.mb); free_buf(l.coff); free_buf(l.mtfp);
      free_buf(l.hdr); free_buf(l.poff); free_buf(l.pcpos); free_buf(l.pcsrc); free_buf(l.pctfp);
      free_buf(l.phdr); free_ev(l.freed); free_ev(l.planned);
    }
    for (auto& p : s.plans) {
      free_buf(p.off); free_buf(p.cpos); free_buf(p.csrc); free_buf(p.ctfp);
      free_buf(p.hdr); free_ev(p.ready); free_ev(p.freed);
    }
    for (auto& q : s.queues) {
      free_buf(q.q);
      free_buf(q.rq);
      free_buf(q.state);
    }
  }
  for (auto& t : c->ts) {
    free_buf(t.flag); free_buf(t.agg); free_buf(t.inc);
  }
  free_buf(c->code); free_buf(c->selftest); free_buf(c->x_mb); free_buf(c->x_coff); free_buf(c->x_mtfp); free_buf(c->x_hdr);
  for (DevBuf* b : {&c->pb_key[0], &c->pb_key[1], &c->pb_val[0], &c->pb_val[1], &c->pb_child,
                    &c->pb_hist, &c->pb_dtot, &c->pb_first, &c->pb_endp, &c->pb_hsz, &c->pb_left,
                    &c->pb_hoff, &c->pb_rem})
    free_buf(*b);
  free_ev(c->fork); free_ev(c->x_planned); free_ev(c->join_plan); free_ev(c->join_copy);
  for (int k = 0; k < FIN_STREAMS; ++k) {
    free_ev(c->fin_fork[k]);
    free_ev(c->fin_join[k]);
    if (c->own_fin[k]) cudaStreamDestroy(c->own_fin[k]);
  }
  free_ev(c->fin_plan); free_ev(c->copy_done);
  for (cudaEvent_t e : c->prof.pool) cudaEventDestroy(e);
  for (auto& t : c->ts_call) {
    free_buf(t.flag); free_buf(t.agg); free_buf(t.inc);
  }
  for (auto& e : c->call_fork) free_ev(e);
  for (auto& e : c->call_join) free_ev(e);
  free_scalars(c);
  delete c;
  return RO_OK;
}

ro_status ro_ctx_reset(ro_ctx* c) {
  if (!c) return RO_E_INVAL;
  DeviceGuard g(c->device);
  RO_TRY(join(c));   // the next expansion reuses buffers the other streams may still read
  c->exps.clear();
  c->err.clear();
  return RO_OK;
}

ro_status ro_ctx_set_streams(ro_ctx* c, void* plan_stream, void* copy_stream) {
  RO_TRY(enter(c));
  DeviceGuard g(c->device);
  RO_TRY(join(c));
  c->plan_stream = plan_stream ? (cudaStream_t)plan_stream : c->stream;
  c->copy_stream = copy_stream ? (cudaStream_t)copy_stream : c->stream;
  // with streams of its own for assembly, the context also runs the
  // completion lists and plans on FIN_STREAMS streams of its own, so a
  // commit's plan overlaps the next commits' scatters and plans
  if (c->plan_stream != c->stream) {
    for (int k = 0; k < FIN_STREAMS; ++k) {
      if (!c->own_fin[k]) {
        cudaError_t e = cudaStreamCreateWithFlags(&c->own_fin[k], cudaStreamNonBlocking);
        if (e != cudaSuccess) {
          c->own_fin[k] = nullptr;
          return cuda_fail(c, e, "cudaStreamCreate");
        }
      }
      c->fin_stream[k] = c->own_fin[k];
    }
  } else {
    for (auto& f : c->fin_stream) f = c->stream;
  }
  c->Lp.stream = c->plan_stream;
  c->Lc.stream = c->copy_stream;
  for (int k = 0; k < FIN_STREAMS; ++k) c->Lf[k].stream = c->fin_stream[k];
  return RO_OK;
}

ro_status ro_ctx_set_call_streams(ro_ctx* c, void* const* streams, uint32_t n) {
  RO_TRY(enter(c));
  if (n > c->n_calls) return fail(c, RO_E_INVAL, "ro_ctx_set_call_streams: %u streams for %u Calls", n, c->n_calls);
  if (n && !streams) return fail(c, RO_E_INVAL, "ro_ctx_set_call_streams: NULL stream list");
  DeviceGuard g(c->device);
  RO_TRY(join(c));   // pending admissions on the old streams first
  for (uint32_t k = 0; k < c->n_calls; ++k)
    c->call_stream[k] = (k < n && streams[k]) ? (cudaStream_t)streams[k] : c->stream;
  return RO_OK;
}

ro_status ro_ctx_join(ro_ctx* c) {
  RO_TRY(enter(c));
  DeviceGuard g(c->device);
  return join(c);
}

ro_status ro_ctx_sync(ro_ctx* c) {
  RO_TRY(enter(c));
  DeviceGuard g(c->device);
  return sync_and_check(c);
}

ro_status ro_ctx_stats(ro_ctx* c, ro_stats* out) {
  RO_TRY(enter(c));
  if (!out) return fail(c, RO_E_INVAL, "stats output is NULL");
  DeviceGuard g(c->device);
  ro_status st = sync_and_check(c);
  uint64_t* o = &out->accepted;
  for (int k = 0; k < 13; ++k) o[k] = c->hs->stats[k];
  return st;
}

const char* ro_last_error(const ro_ctx* c) { return c ? c->err.c_str() : "no context"; }

ro_status ro_ctx_profile(ro_ctx* c, uint32_t kernel_mask) {
  RO_TRY(enter(c));
  c->prof.mask = kernel_mask & ((1u << K_COUNT) - 1u);
  return RO_OK;
}

ro_status ro_ctx_profile_read(ro_ctx* c, uint64_t* launches, uint64_t* timed, double* ms,
                              uint32_t n_kernels) {
  RO_TRY(enter(c));
  DeviceGuard g(c->device);
  RO_TRY(join(c));
  cudaError_t e = cudaStreamSynchronize(c->stream);
  if (e != cudaSuccess) return cuda_fail(c, e, "synchronise");
  Profiler& p = c->prof;
  for (const auto& m : p.marks) {
    float t = 0.f;
    if (cudaEventElapsedTime(&t, p.pool[m.second], p.pool[m.second + 1]) == cudaSuccess) {
      p.ms[m.first] += t;
      p.timed[m.first] += 1;
    } else {
      cudaGetLastError();
    }
  }
  p.marks.clear();
  p.used = 0;
  const uint32_t k = std::min<uint32_t>(n_kernels, K_COUNT);
  for (uint32_t i = 0; i < k; ++i) {
    if (launches) launches[i] = p.launches[i];
    if (timed) timed[i] = p.timed[i];
    if (ms) ms[i] = p.ms[i];
    p.launches[i] = 0;
    p.timed[i] = 0;
    p.ms[i] = 0.0;
  }
  return RO_OK;
}

// ---------------------------------------------------------------------------
ro_status ro_expand(ro_ctx* c, int32_t parent_xid, const uint32_t* d_counts, uint64_t n_parents,
                    const uint8_t* d_parent_call, uint64_t* d_offsets, uint32_t* d_child_parent,
                    uint32_t* d_child_ordinal, uint64_t child_cap, uint32_t* d_empty_parents,
                    uint64_t* h_n_children, uint64_t* h_n_empty, int32_t* xid) {
  RO_TRY(enter(c));
  if (!xid || !h_n_children || !d_offsets || (n_parents && !d_counts))
    return fail(c, RO_E_INVAL, "ro_expand: NULL argument");
  if (n_parents >= (1ull << 32)) return fail(c, RO_E_OVERFLOW, "ro_expand: 2^32 parents or more");
  if ((int)c->exps.size() >= MAX_EXPANSIONS)
    return fail(c, RO_E_STATE, "ro_expand: more than %d expansions in one context", MAX_EXPANSIONS);
  if (parent_xid != -1) {
    Expansion* px = get_exp(c, parent_xid);
    if (!px) return fail(c, RO_E_STATE, "ro_expand: unknown parent expansion %d", parent_xid);
    if (px->N != n_parents)
      return fail(c, RO_E_INVAL, "ro_expand: %llu parents but parent expansion has %llu children",
                  (unsigned long long)n_parents, (unsigned long long)px->N);
  }
  DeviceGuard g(c->device);
  RO_TRY(settle_calls(c));   // after the Calls' pending admissions
  const size_t slot = c->exps.size();
  if (c->slots.size() <= slot) c->slots.resize(slot + 1);
  ExpSlot& S = c->slots[slot];
  const uint64_t P = n_parents;
  const uint64_t cap_children = std::min<uint64_t>(child_cap, (1ull << 32));
  const uint64_t tfp_entries = ceil_div(cap_children, FILL_TILE) + 1;
  RO_TRY(ensure(c, S.offsets, (P + 1) * sizeof(uint64_t), "offsets"));
  RO_TRY(ensure(c, S.pw, P * sizeof(uint64_t), "parent counters"));
  RO_TRY(ensure(c, S.tfp, tfp_entries * sizeof(uint32_t), "fill tiles"));
  ExpandScanArgs sa{};
  sa.counts = d_counts;
  sa.P = P;
  sa.offsets_user = d_offsets;
  sa.offsets = (uint64_t*)S.offsets.p;
  sa.pw = (unsigned long long*)S.pw.p;
  sa.empty_out = d_empty_parents;
  sa.tfp = (uint32_t*)S.tfp.p;
  sa.tfp_cap = tfp_entries;
  sa.ds = c->ds;
  RO_TRY(tile_status(c, TS_EXPAND, ceil_div(P, (uint64_t)EXP_THREADS * EXP_ITEMS), &sa.ts));
  cudaMemsetAsync(&c->ds->n_heavy, 0, sizeof(unsigned long long), c->stream);
  launch_expand_scan(c->L, sa);
  RO_TRY(check_launch(c, "expand_scan"));
  RO_TRY(sync_and_check(c));
  const uint64_t N = c->hs->n_children;
  *h_n_children = N;
  if (h_n_empty) *h_n_empty = c->hs->n_empty;
  if (N >= (1ull << 32)) return fail(c, RO_E_OVERFLOW, "ro_expand: 2^32 children or more");
  if (N > child_cap)
    return fail(c, RO_E_CAPACITY, "ro_expand: %llu children exceed child_cap %llu",
                (unsigned long long)N, (unsigned long long)child_cap);
  if (N && (!d_child_parent || !d_child_ordinal))
    return fail(c, RO_E_INVAL, "ro_expand: NULL child arrays");

  const uint64_t mtfp_cap = ceil_div(N, AM_TILE) + 2;
  RO_TRY(ensure(c, S.slot, N * sizeof(Slot), "child slots"));
  RO_TRY(ensure(c, S.par, N * sizeof(uint32_t), "child parents"));
  RO_TRY(ensure(c, S.bitmap, BM_SLOTS * ceil_div(P, 32) * sizeof(uint32_t), "completion bitmaps"));
  RO_TRY(ensure(c, S.gb, P * sizeof(unsigned long long), "GroupFailure barriers"));
  for (auto& l : S.lists) {
    RO_TRY(ensure(c, l.done, P * sizeof(uint32_t), "completed parents"));
    RO_TRY(ensure(c, l.status, P, "completed parents"));
    RO_TRY(ensure(c, l.mb, (P + 1) * sizeof(uint32_t), "member bases"));
    RO_TRY(ensure(c, l.coff, P * sizeof(uint32_t), "member bases"));
    RO_TRY(ensure(c, l.mtfp, mtfp_cap * sizeof(uint32_t), "member tiles"));
    RO_TRY(ensure(c, l.hdr, sizeof(ListHdr), "list header"));
    RO_TRY(ensure(c, l.poff, (P + 1) * sizeof(uint64_t), "assembly plan"));
    RO_TRY(ensure(c, l.pcpos, N * sizeof(uint64_t), "assembly plan"));
    RO_TRY(ensure(c, l.pcsrc, N * sizeof(uint64_t), "assembly plan"));
    RO_TRY(ensure(c, l.phdr, sizeof(PlanHdr), "assembly plan"));
  }
  for (auto& p : S.plans) {
    RO_TRY(ensure(c, p.off, (P + 1) * sizeof(uint64_t), "assembly plan"));
    RO_TRY(ensure(c, p.cpos, N * sizeof(uint64_t), "assembly plan"));
    RO_TRY(ensure(c, p.csrc, N * sizeof(uint64_t), "assembly plan"));
    RO_TRY(ensure(c, p.hdr, sizeof(PlanHdr), "assembly plan"));
  }
  cudaMemsetAsync(S.bitmap.p, 0, BM_SLOTS * ceil_div(P, 32) * sizeof(uint32_t), c->stream);
  cudaMemsetAsync(S.gb.p, 0, P * sizeof(unsigned long long), c->stream);   // no barrier (commit 0)
  ExpandFillArgs fa{};
  fa.offsets = (const uint64_t*)S.offsets.p;
  fa.P = P;
  fa.N = N;
  fa.tfp = (const uint32_t*)S.tfp.p;
  fa.parent_call = d_parent_call;
  fa.child_parent = d_child_parent;
  fa.child_ordinal = d_child_ordinal;
  fa.slot = (Slot*)S.slot.p;
  fa.par = (uint32_t*)S.par.p;
  launch_expand_fill(c->L, fa);
  RO_TRY(check_launch(c, "expand_fill"));
  if (S.queues.size() < c->n_calls) S.queues.resize(c->n_calls);
  for (auto& q : S.queues) q.ready = false;

  Expansion x;
  x.parent_xid = parent_xid;
  x.P = P;
  x.N = N;
  x.heavy = c->hs->n_heavy != 0 && 4 * c->hs->n_heavy >= x.N;
  c->exps.push_back(x);
  *xid = (int32_t)slot;
  return RO_OK;
}

// ---------------------------------------------------------------------------
// The admission arguments of one Call (queue, scan slot, outputs).
ro_status ready_args(ro_ctx* c, int32_t xid, uint32_t call, const uint32_t* d_cand, uint64_t n_cand,
                     uint32_t batch_size, int32_t flush, uint32_t* d_batched, uint64_t batched_cap,
                     uint64_t* d_n_batched, ReadyArgs* out) {
  Expansion* x = get_exp(c, xid);
  ExpSlot& S = c->slots[xid];
  QueueBufs& Q = S.queues[call];
  RO_TRY(queue_ready(c, Q, x->N));
  ReadyArgs ra{};
  ra.cand = d_cand;
  ra.n_cand = d_cand ? n_cand : x->N;
  ra.N = x->N;
  ra.slot = (Slot*)S.slot.p;
  ra.check_call = c->n_calls > 1;
  ra.call = call;
  ra.batch_size = batch_size;
  ra.flush = flush != 0;
  ra.cap = batched_cap;
  ra.queue = (uint32_t*)Q.q.p;
  ra.qstate = (unsigned long long*)Q.state.p;
  ra.rq = (const uint32_t*)Q.rq.p;
  ra.batched = d_batched;
  ra.n_batched_out = d_n_batched;
  ra.ds = c->ds;
  ra.rs = c->rs + call;
  RO_TRY(tile_status_buf(c, c->ts_call[call], ceil_div(ra.n_cand, (uint64_t)RB_THREADS * RB_ITEMS),
                         &ra.ts));
  *out = ra;
  return RO_OK;
}

ro_status ro_batch_ready(ro_ctx* c, int32_t xid, uint32_t call, const uint32_t* d_cand,
                         uint64_t n_cand, uint32_t batch_size, int32_t flush, uint32_t* d_batched,
                         uint64_t batched_cap, uint64_t* d_n_batched, uint64_t* h_n_batched,
                         uint64_t* h_n_batches) {
  RO_TRY(enter(c));
  Expansion* x = get_exp(c, xid);
  if (!x) return fail(c, RO_E_STATE, "ro_batch_ready: unknown expansion %d", xid);
  if (call >= c->n_calls) return fail(c, RO_E_INVAL, "ro_batch_ready: call %u out of range", call);
  if (batch_size == 0) return fail(c, RO_E_INVAL, "ro_batch_ready: batch_size is 0");
  if (batched_cap && !d_batched) return fail(c, RO_E_INVAL, "ro_batch_ready: NULL d_batched");
  if (d_cand && n_cand > MAX_CAND)
    return fail(c, RO_E_INVAL, "ro_batch_ready: more than 2^30-2 candidates in one call");
  DeviceGuard g(c->device);
  ReadyArgs ra{};
  RO_TRY(ready_args(c, xid, call, d_cand, n_cand, batch_size, flush, d_batched, batched_cap,
                    d_n_batched, &ra));
  for (cudaStream_t s : c->call_stream) ra.calls_concurrent |= (s != c->stream);
  ra.calls_concurrent &= ra.check_call;
  // on the Call's stream when it has one, after everything issued on the
  // context's stream so far; the context's stream waits for it before its
  // next launch
  LaunchCfg Lr = c->L;
  const cudaStream_t cs = c->call_stream[call];
  if (cs != c->stream) {
    RO_TRY(order(c, c->call_fork[call], c->stream, cs));
    Lr.stream = cs;
  }
  launch_ready(Lr, ra);
  RO_TRY(check_launch(c, "batch_ready"));
  if (cs != c->stream) c->call_pending[call] = 1;
  if (h_n_batched || h_n_batches) {
    ro_status st = sync_and_check(c);
    cudaError_t e = cudaMemcpyAsync(c->hrs + call, c->rs + call, sizeof(ReadyScalars),
                                    cudaMemcpyDeviceToHost, c->stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(c->stream);
    if (e != cudaSuccess) return cuda_fail(c, e, "synchronise");
    if (h_n_batched) *h_n_batched = c->hrs[call].rb_npop;
    if (h_n_batches) *h_n_batches = c->hrs[call].rb_n_batches;
    return st;
  }
  return RO_OK;
}

// ---------------------------------------------------------------------------
ro_status ro_batch_ready_calls(ro_ctx* c, int32_t xid, uint32_t n, const uint32_t* calls,
                               const uint32_t* d_cand, uint64_t n_cand, uint32_t batch_size,
                               int32_t flush, uint32_t* const* d_batched,
                               const uint64_t* batched_cap, uint64_t* const* d_n_batched) {
  RO_TRY(enter(c));
  const char* fn = "ro_batch_ready_calls";
  Expansion* x = get_exp(c, xid);
  if (!x) return fail(c, RO_E_STATE, "%s: unknown expansion %d", fn, xid);
  if (n == 0 || n > RB_CALLS_MAX) return fail(c, RO_E_INVAL, "%s: %u Calls (1 to %u)", fn, n, RB_CALLS_MAX);
  if (!calls || !d_batched || !batched_cap) return fail(c, RO_E_INVAL, "%s: NULL argument", fn);
  if (batch_size == 0) return fail(c, RO_E_INVAL, "%s: batch_size is 0", fn);
  if (d_cand && n_cand > MAX_CAND)
    return fail(c, RO_E_INVAL, "%s: more than 2^30-2 candidates in one call", fn);
  for (uint32_t k = 0; k < n; ++k) {
    if (calls[k] >= c->n_calls) return fail(c, RO_E_INVAL, "%s: call %u out of range", fn, calls[k]);
    if (batched_cap[k] && !d_batched[k]) return fail(c, RO_E_INVAL, "%s: NULL d_batched", fn);
    for (uint32_t j = 0; j < k; ++j)
      if (calls[j] == calls[k]) return fail(c, RO_E_INVAL, "%s: call %u named twice", fn, calls[k]);
  }
  DeviceGuard g(c->device);
  RO_TRY(settle_calls(c));   // after the Calls' pending admissions on their streams
  MultiReadyArgs m{};
  m.n = n;
  for (uint32_t k = 0; k < n; ++k)
    RO_TRY(ready_args(c, xid, calls[k], d_cand, n_cand, batch_size, flush, d_batched[k], batched_cap[k],
                      d_n_batched ? d_n_batched[k] : nullptr, &m.a[k]));
  const uint64_t per = ceil_div(m.a[0].n_cand, (uint64_t)RB_THREADS * RB_ITEMS) + 1;
  if (per * n <= (uint64_t)c->L.grid_rb_coop_calls) {
    launch_ready_calls(c->L, m);
  } else {   // too long a list for one grid: one admission after another
    for (uint32_t k = 0; k < n; ++k) launch_ready(c->L, m.a[k]);
  }
  return check_launch(c, "batch_ready_calls");
}

// ---------------------------------------------------------------------------
ro_status ro_ctx_selftest_timeout(ro_ctx* c, uint32_t kind) {
  RO_TRY(enter(c));
  if (kind > 1) return fail(c, RO_E_INVAL, "ro_ctx_selftest_timeout: kind %u (0 or 1)", kind);
  DeviceGuard g(c->device);
  RO_TRY(sync_and_check(c));   // earlier work settled, its errors reported first
  const size_t flags = 2 * sizeof(unsigned long long), vals = 2 * 16;
  RO_TRY(ensure(c, c->selftest, flags + 2 * vals + sizeof(ReadyScalars), "self-test scratch"));
  char* base = (char*)c->selftest.p;
  cudaError_t e = cudaMemsetAsync(base, 0, flags + 2 * vals + sizeof(ReadyScalars), c->stream);
  if (e != cudaSuccess) return cuda_fail(c, e, "self-test scratch");
  SelftestArgs a{};
  a.kind = kind;
  a.ts.flag = (unsigned long long*)base;
  a.ts.agg = (unsigned long long*)(base + flags);
  a.ts.inc = (unsigned long long*)(base + flags + vals);
  a.epoch = 1ull;   // the zeroed flags hold epoch 0
  a.rs = (ReadyScalars*)(base + flags + 2 * vals);
  a.err = &c->ds->err;
  launch_selftest(c->stream, a);
  RO_TRY(check_launch(c, "selftest"));
  return sync_and_check(c);
}

// ---------------------------------------------------------------------------
ro_status ro_batch_ready_parent(ro_ctx* c, int32_t xid, uint32_t call, const uint32_t* d_cand,
                                uint64_t n_cand, uint32_t batch_size, int32_t flush,
                                uint32_t* d_batched, uint64_t batched_cap, uint64_t* d_batch_off,
                                uint64_t batch_off_cap, uint64_t* d_n_batched,
                                uint64_t* d_n_batches, uint64_t* h_n_batched,
                                uint64_t* h_n_batches) {
  RO_TRY(enter(c));
  Expansion* x = get_exp(c, xid);
  const char* fn = "ro_batch_ready_parent";
  if (!x) return fail(c, RO_E_STATE, "%s: unknown expansion %d", fn, xid);
  if (call >= c->n_calls) return fail(c, RO_E_INVAL, "%s: call %u out of range", fn, call);
  if (batch_size == 0) return fail(c, RO_E_INVAL, "%s: batch_size is 0", fn);
  if (batched_cap && !d_batched) return fail(c, RO_E_INVAL, "%s: NULL d_batched", fn);
  if (d_cand && n_cand > MAX_CAND)
    return fail(c, RO_E_INVAL, "%s: more than 2^30-2 candidates in one call", fn);
  DeviceGuard g(c->device);
  RO_TRY(settle_calls(c));   // after the Calls' pending admissions
  ExpSlot& S = c->slots[xid];
  QueueBufs& Q = S.queues[call];
  RO_TRY(queue_ready(c, Q, x->N));
  const uint64_t N = x->N, P = x->P, tiles = std::max<uint64_t>(1, ceil_div(N, (uint64_t)PB_TILE));
  const size_t n4 = std::max<uint64_t>(N, 1) * sizeof(uint32_t);
  for (DevBuf* b : {&c->pb_key[0], &c->pb_key[1], &c->pb_val[0], &c->pb_val[1], &c->pb_child,
                    &c->pb_hsz, &c->pb_hoff, &c->pb_rem})
    RO_TRY(ensure(c, *b, n4, "parent-bound scratch"));
  RO_TRY(ensure(c, c->pb_left, std::max<uint64_t>(N, 1), "parent-bound scratch"));
  RO_TRY(ensure(c, c->pb_hist, PB_DIGITS * tiles * sizeof(uint32_t), "parent-bound histogram"));
  RO_TRY(ensure(c, c->pb_dtot, PB_DIGITS * sizeof(uint32_t), "parent-bound digit totals"));
  RO_TRY(ensure(c, c->pb_first, std::max<uint64_t>(P, 1) * sizeof(uint32_t), "parent-bound ranges"));
  RO_TRY(ensure(c, c->pb_endp, std::max<uint64_t>(P, 1) * sizeof(uint32_t), "parent-bound ranges"));

  ReadyArgs ra{};
  ra.cand = d_cand;
  ra.n_cand = d_cand ? n_cand : N;
  ra.N = N;
  ra.slot = (Slot*)S.slot.p;
  ra.check_call = c->n_calls > 1;
  ra.call = call;
  ra.batch_size = batch_size;
  ra.flush = flush != 0;
  ra.cap = batched_cap;
  ra.queue = (uint32_t*)Q.q.p;
  ra.qstate = (unsigned long long*)Q.state.p;
  ra.rq = (const uint32_t*)Q.rq.p;
  ra.batched = d_batched;
  ra.n_batched_out = nullptr;
  ra.parent_bound = 1;
  ra.ds = c->ds;
  ra.rs = c->rs + call;
  RO_TRY(tile_status_buf(c, c->ts_call[call], ceil_div(ra.n_cand, (uint64_t)RB_THREADS * RB_ITEMS),
                         &ra.ts));

  ParentArgs pa{};
  pa.N = N;
  pa.P = P;
  pa.B = batch_size;
  pa.flush = flush != 0;
  int bits = 0;
  while (bits < 32 && P > 1 && ((P - 1) >> bits) != 0) ++bits;
  pa.passes = (bits + 7) / 8;
  pa.par = (const uint32_t*)S.par.p;
  pa.slot = (Slot*)S.slot.p;
  pa.queue = (uint32_t*)Q.q.p;
  pa.qstate = (unsigned long long*)Q.state.p;
  pa.batched = d_batched;
  pa.cap = batched_cap;
  pa.batch_off = d_batch_off;
  pa.off_cap = batch_off_cap;
  pa.n_batched_out = d_n_batched;
  pa.n_batches_out = d_n_batches;
  for (int k = 0; k < 2; ++k) {
    pa.key[k] = (uint32_t*)c->pb_key[k].p;
    pa.val[k] = (uint32_t*)c->pb_val[k].p;
  }
  pa.child = (uint32_t*)c->pb_child.p;
  pa.hist = (uint32_t*)c->pb_hist.p;
  pa.dtot = (uint32_t*)c->pb_dtot.p;
  pa.first = (uint32_t*)c->pb_first.p;
  pa.endp = (uint32_t*)c->pb_endp.p;
  pa.hsz = (uint32_t*)c->pb_hsz.p;
  pa.left = (uint8_t*)c->pb_left.p;
  pa.hoff = (uint32_t*)c->pb_hoff.p;
  pa.rem = (uint32_t*)c->pb_rem.p;
  pa.ds = c->ds;
  RO_TRY(tile_status(c, TS_PARENT, tiles, &pa.ts));

  launch_ready(c->L, ra);
  launch_parent(c->L, pa);
  RO_TRY(check_launch(c, "batch_ready_parent"));
  if (h_n_batched || h_n_batches) {
    ro_status st = sync_and_check(c);
    if (h_n_batched) *h_n_batched = c->hs->pb_npop;
    if (h_n_batches) *h_n_batches = c->hs->pb_nb;
    return st;
  }
  return RO_OK;
}

// ---------------------------------------------------------------------------
ro_status ro_retry(ro_ctx* c, int32_t xid, uint32_t call, const uint32_t* d_children, uint64_t n,
                   uint64_t* h_n_retried) {
  RO_TRY(enter(c));
  Expansion* x = get_exp(c, xid);
  if (!x) return fail(c, RO_E_STATE, "ro_retry: unknown expansion %d", xid);
  if (call >= c->n_calls) return fail(c, RO_E_INVAL, "ro_retry: call %u out of range", call);
  if (n && !d_children) return fail(c, RO_E_INVAL, "ro_retry: NULL d_children");
  if (n >= 0xFFFFFFFFull) return fail(c, RO_E_OVERFLOW, "ro_retry: 2^32-1 entries or more");
  DeviceGuard g(c->device);
  RO_TRY(settle_calls(c));   // after the Calls' pending admissions
  ExpSlot& S = c->slots[xid];
  if (h_n_retried) *h_n_retried = 0;
  if (n == 0) return RO_OK;
  QueueBufs& Q = S.queues[call];
  RO_TRY(queue_ready(c, Q, x->N));
  RetryArgs ta{};
  ta.children = d_children;
  ta.n = n;
  ta.N = x->N;
  ta.slot = (Slot*)S.slot.p;
  ta.check_call = c->n_calls > 1;
  ta.call = call;
  ta.rq = (uint32_t*)Q.rq.p;
  ta.qstate = (unsigned long long*)Q.state.p;
  ta.ds = c->ds;
  RO_TRY(tile_status(c, TS_RETRY, ceil_div(n, (uint64_t)RT_THREADS * RT_ITEMS), &ta.ts));
  launch_retry(c->L, ta);
  RO_TRY(check_launch(c, "retry"));
  if (h_n_retried) {
    ro_status st = sync_and_check(c);
    *h_n_retried = c->hs->rt_done;
    return st;
  }
  return RO_OK;
}

// ---------------------------------------------------------------------------
ro_status ro_gather_commit(ro_ctx* c, int32_t xid, uint64_t n, const uint64_t* d_n,
                           const uint32_t* d_child, const uint8_t* d_state, const uint32_t* d_len,
                           const uint64_t* d_arena_off, const uint32_t* d_gen, uint64_t arena_bytes,
                           uint8_t* d_code, uint32_t* d_done_parents, uint64_t done_cap,
                           uint64_t* d_n_done, uint64_t* h_n_done) {
  RO_TRY(enter(c));
  Expansion* x = get_exp(c, xid);
  if (!x) return fail(c, RO_E_STATE, "ro_gather_commit: unknown expansion %d", xid);
  if (n >= (1ull << 32)) return fail(c, RO_E_OVERFLOW, "ro_gather_commit: 2^32 reports or more");
  if (n && (!d_child || !d_state || !d_len || !d_arena_off))
    return fail(c, RO_E_INVAL, "ro_gather_commit: NULL report array");
  if (arena_bytes >= MAX_ARENA) return fail(c, RO_E_OVERFLOW, "ro_gather_commit: arena of 2^48 bytes or more");
  if (d_done_parents && done_cap < std::min<uint64_t>(n, x->P))
    return fail(c, RO_E_INVAL, "ro_gather_commit: done_cap below min(n, parents)");
  DeviceGuard g(c->device);
  RO_TRY(settle_calls(c));   // after the Calls' pending admissions
  ExpSlot& S = c->slots[xid];
  const int ls = (int)(x->commits % RING);
  ListSlot& LS = S.lists[ls];
  CommitArgs ca{};
  ca.n_host = n;
  ca.d_n = d_n;
  ca.child = d_child;
  ca.state = d_state;
  ca.len = d_len;
  ca.off = d_arena_off;
  ca.gen = d_gen;
  ca.arena_bytes = arena_bytes;
  ca.N = x->N;
  ca.P = x->P;
  ca.slot = (Slot*)S.slot.p;
  ca.par = (const uint32_t*)S.par.p;
  ca.pw = (unsigned long long*)S.pw.p;
  const int bs = (int)(x->commits % BM_SLOTS);   // bitmap slot of this commit
  const uint64_t n_words = ceil_div(x->P, 32);
  ca.bitmap = (uint32_t*)S.bitmap.p + bs * n_words;
  ca.heavy = x->heavy ? 1 : 0;
  ca.tfp = (const uint32_t*)S.tfp.p;
  ca.n_fill_tiles = ceil_div(x->N, FILL_TILE);
  ca.gb = (unsigned long long*)S.gb.p;
  if (++c->commit_seq == 0) {   // wrapped: old tags could look current again
    for (auto& sl : c->slots)
      if (sl.gb.p) cudaMemsetAsync(sl.gb.p, 0, sl.gb.cap, c->stream);
    c->commit_seq = 1;
  }
  ca.seq = c->commit_seq;   // from 1: 0 in the barrier table means no barrier
  if (d_code) {
    ca.code = d_code;
  } else {
    RO_TRY(ensure(c, c->code, n, "report verdicts"));
    ca.code = (uint8_t*)c->code.p;
  }
  ca.done_user = d_done_parents;
  ca.done_int = (uint32_t*)LS.done.p;
  ca.n_done_out = d_n_done;
  ca.offsets = (const uint64_t*)S.offsets.p;
  ca.list = list_bufs(LS, ceil_div(x->N, AM_TILE) + 2);
  // the chunk table of the plan: one entry per 16 KB of the arena the
  // reports reference (a plan that needs more makes the copy search instead)
  const uint64_t want_chunks = std::min<uint64_t>(ceil_div(arena_bytes, AC_CHUNK) + 2, 1ull << 31);
  if (LS.pctfp_cap < want_chunks) {
    RO_TRY(ensure(c, LS.pctfp, want_chunks * sizeof(uint32_t), "chunk table"));
    LS.pctfp_cap = LS.pctfp.cap / sizeof(uint32_t);
  }
  ca.plan = list_plan_bufs(LS, std::max<uint64_t>(x->N, 1));
  ca.ds = c->ds;
  // consecutive commits plan on the completion streams in turn, each with a
  // scan slot of its own; every slot is sized together, so that a capture of
  // later commits finds its slot grown whichever stream the first calls took
  const int pf = (int)(c->commit_seq % FIN_STREAMS);
  ca.pslot = pf;
  for (int k = 0; k < FIN_STREAMS; ++k) {
    TileStatus<Quad64> t;
    RO_TRY(tile_status(c, commit_slot(k), ceil_div(ceil_div(x->P, 32), (uint64_t)CP_WORDS), &t));
    if (k == pf) ca.tsq = t;
  }
  // The bitmap slots of this commit and the next BM_WAIT - 1 are free once
  // every plan up to commit w - BM_WAIT - 1 is done: wait for the latest such
  // plan of each completion stream (a stream runs its plans in order).
  if (x->commits % BM_WAIT == 0 && x->commits > (uint64_t)BM_WAIT) {
    const uint64_t w = x->commits;
    bool seen[FIN_STREAMS] = {};
    int n_seen = 0;
    // (commits w - BM_SLOTS .. w - BM_WAIT - 1: the slot of commit w - BM_SLOTS
    // is this commit's, and its event is not overwritten yet)
    for (uint64_t j = w - BM_WAIT - 1; j + BM_SLOTS >= w && n_seen < FIN_STREAMS; --j) {
      const int k = S.bm_stream[j % BM_SLOTS];
      if (!seen[k]) {
        RO_TRY(ev_wait(c, S.bm_free[j % BM_SLOTS], c->stream));
        seen[k] = true;
        ++n_seen;
      }
      if (j == 0) break;
    }
  }
  launch_commit_scatter(c->L, ca);
  // the completed list and its plan follow the scatter (on their own stream
  // when the context has one); the list slot is free once the assembly that
  // read it (RING commits ago) is done
  const cudaStream_t fs = c->fin_stream[pf];
  RO_TRY(order(c, c->fin_fork[pf], c->stream, fs));
  RO_TRY(ev_wait(c, LS.freed, fs));
  RO_TRY(ev_wait(c, LS.planned, fs));
  launch_commit_plan(c->Lf[pf], ca);
  if (fs != c->stream) {
    RO_TRY(ev_record(c, S.bm_free[bs], fs));
    S.bm_stream[bs] = pf;
    RO_TRY(ev_record(c, LS.planned, fs));
  }
  c->last_fin = pf;
  RO_TRY(check_launch(c, "gather_commit"));
  x->last_list = ls;
  x->commits += 1;
  if (h_n_done) {
    ro_status st = sync_and_check(c);
    *h_n_done = c->hs->cm_n_done[pf];
    return st;
  }
  return RO_OK;
}

// ---------------------------------------------------------------------------
namespace {
struct ElemOut {
  uint64_t* base;
  uint8_t* state;
  uint64_t* off;
  uint32_t* len;
  uint64_t cap;
  uint64_t* d_n;
  uint64_t* h_n;
};
ro_status assemble_impl(ro_ctx* c, int32_t xid, const uint8_t* d_arena, uint64_t arena_bytes,
                        const uint32_t* d_parents, uint64_t n_parents, const uint64_t* d_n_parents,
                        uint8_t* d_status, uint64_t* d_out_off, uint32_t* d_out_len, uint8_t* d_out,
                        uint64_t out_cap, uint64_t* d_out_cursor, uint64_t* d_out_bytes,
                        uint64_t* h_out_bytes, const ElemOut* eo);
}  // namespace

ro_status ro_assemble(ro_ctx* c, int32_t xid, const uint8_t* d_arena, uint64_t arena_bytes,
                      const uint32_t* d_parents, uint64_t n_parents, const uint64_t* d_n_parents,
                      uint8_t* d_status, uint64_t* d_out_off, uint32_t* d_out_len, uint8_t* d_out,
                      uint64_t out_cap, uint64_t* d_out_cursor, uint64_t* d_out_bytes,
                      uint64_t* h_out_bytes) {
  return assemble_impl(c, xid, d_arena, arena_bytes, d_parents, n_parents, d_n_parents, d_status,
                       d_out_off, d_out_len, d_out, out_cap, d_out_cursor, d_out_bytes, h_out_bytes,
                       nullptr);
}

ro_status ro_assemble_list(ro_ctx* c, int32_t xid, const uint8_t* d_arena, uint64_t arena_bytes,
                           const uint32_t* d_parents, uint64_t n_parents,
                           const uint64_t* d_n_parents, uint8_t* d_status, uint64_t* d_out_off,
                           uint32_t* d_out_len, uint8_t* d_out, uint64_t out_cap,
                           uint64_t* d_out_cursor, uint64_t* d_out_bytes, uint64_t* h_out_bytes,
                           uint64_t* d_elem_base, uint8_t* d_elem_state, uint64_t* d_elem_off,
                           uint32_t* d_elem_len, uint64_t elem_cap, uint64_t* d_n_elems,
                           uint64_t* h_n_elems) {
  RO_TRY(enter(c));
  if (!d_elem_base || (elem_cap && (!d_elem_state || !d_elem_off || !d_elem_len)))
    return fail(c, RO_E_INVAL, "ro_assemble_list: NULL list-structure output");
  const ElemOut eo{d_elem_base, d_elem_state, d_elem_off, d_elem_len, elem_cap, d_n_elems, h_n_elems};
  return assemble_impl(c, xid, d_arena, arena_bytes, d_parents, n_parents, d_n_parents, d_status,
                       d_out_off, d_out_len, d_out, out_cap, d_out_cursor, d_out_bytes, h_out_bytes,
                       &eo);
}

ro_status ro_filter_reports(ro_ctx* c, uint8_t* d_state, const uint8_t* d_keep, uint64_t n) {
  RO_TRY(enter(c));
  if (n && (!d_state || !d_keep)) return fail(c, RO_E_INVAL, "ro_filter_reports: NULL argument");
  if (!n) return RO_OK;
  DeviceGuard g(c->device);
  launch_filter(c->stream, d_state, d_keep, n, c->num_sms * 8);
  return check_launch(c, "filter_reports");
}

}  // extern "C"

namespace {
ro_status assemble_impl(ro_ctx* c, int32_t xid, const uint8_t* d_arena, uint64_t arena_bytes,
                        const uint32_t* d_parents, uint64_t n_parents, const uint64_t* d_n_parents,
                        uint8_t* d_status, uint64_t* d_out_off, uint32_t* d_out_len, uint8_t* d_out,
                        uint64_t out_cap, uint64_t* d_out_cursor, uint64_t* d_out_bytes,
                        uint64_t* h_out_bytes, const ElemOut* eo) {
  RO_TRY(enter(c));
  Expansion* x = get_exp(c, xid);
  if (!x) return fail(c, RO_E_STATE, "ro_assemble: unknown expansion %d", xid);
  if (!d_arena || !d_status || !d_out_off)
    return fail(c, RO_E_INVAL, "ro_assemble: NULL arena, status or offsets");
  if (out_cap && !d_out) return fail(c, RO_E_INVAL, "ro_assemble: NULL output");
  if (!d_parents && x->last_list < 0)
    return fail(c, RO_E_STATE, "ro_assemble: no commit on expansion %d to take parents from", xid);
  if (n_parents >= (1ull << 32)) return fail(c, RO_E_OVERFLOW, "ro_assemble: list of 2^32 or more");
  if (arena_bytes >= MAX_ARENA) return fail(c, RO_E_OVERFLOW, "ro_assemble: arena of 2^48 bytes or more");
  DeviceGuard g(c->device);
  RO_TRY(settle_calls(c));   // after the Calls' pending admissions
  // The arena and the output may be pinned host memory (read and written in
  // place by the copy, no staging copies); pageable host memory is refused.
  int arena_host = 0;
  {
    const uint8_t* dev_arena = nullptr;
    uint8_t* dev_out = nullptr;
    RO_TRY(device_view(c, d_arena, &dev_arena, &arena_host, "arena"));
    int out_host = 0;
    if (d_out) RO_TRY(device_view(c, d_out, &dev_out, &out_host, "output"));
    d_arena = dev_arena;
    d_out = dev_out;
  }
  ExpSlot& S = c->slots[xid];
  const uint64_t member_cap = std::max<uint64_t>(x->N, 1);
  const uint64_t mtfp_cap = ceil_div(member_cap, AM_TILE) + 2;
  // The commit's own list without list structure was planned by the commit
  // (commit_plan): only the copy runs.  Otherwise plan here, into a plan slot.
  const bool planned = !d_parents && !eo;
  PlanSlot& PS = S.plans[x->assembles % RING];
  if (!planned) {
    // chunk table: one entry per 16 KB of output (the copy searches beyond it)
    const uint64_t want_chunks = std::min<uint64_t>(ceil_div(out_cap, AC_CHUNK) + 2, 1ull << 31);
    if (PS.ctfp_cap < want_chunks) {
      RO_TRY(ensure(c, PS.ctfp, want_chunks * sizeof(uint32_t), "chunk table"));
      PS.ctfp_cap = PS.ctfp.cap / sizeof(uint32_t);
    }
  }
  AssembleArgs aa{};
  aa.user_list = d_parents;
  aa.n_host = n_parents;
  aa.d_n = d_parents ? d_n_parents : nullptr;
  aa.P = x->P;
  aa.N = x->N;
  aa.offsets = (const uint64_t*)S.offsets.p;
  aa.pw = (const unsigned long long*)S.pw.p;
  aa.slot = (const Slot*)S.slot.p;
  aa.arena = d_arena;
  aa.arena_bytes = arena_bytes;
  aa.arena_host = arena_host;
  aa.small_chunks = c->copy_small_chunks;
  aa.status = d_status;
  aa.out_off = d_out_off;
  aa.out_len = d_out_len;
  aa.out = d_out;
  aa.out_cap = out_cap;
  aa.cursor = d_out_cursor;
  aa.out_bytes = d_out_bytes;
  if (eo) {
    aa.elem_base = eo->base;
    aa.elem_state = eo->state;
    aa.elem_off = eo->off;
    aa.elem_len = eo->len;
    aa.elem_cap = eo->cap;
    aa.n_elems_out = eo->d_n;
  }
  aa.plan = plan_bufs(PS, member_cap);
  aa.ds = c->ds;
  ListSlot* LS = nullptr;
  if (planned) {
    LS = &S.lists[x->last_list];
    aa.list = list_bufs(*LS, mtfp_cap);
    aa.plan = list_plan_bufs(*LS, member_cap);
    // the copy follows the context's stream (the caller's cursor and
    // outputs) and the commit's plan
    RO_TRY(order(c, c->fork, c->stream, c->copy_stream));
    RO_TRY(order(c, c->fin_plan, c->fin_stream[c->last_fin], c->copy_stream));
  } else if (d_parents) {
    // a caller's list may be longer than the expansion's parents (repeats)
    RO_TRY(ensure(c, PS.off, (n_parents + 1) * sizeof(uint64_t), "assembly plan"));
    aa.plan.off = (uint64_t*)PS.off.p;
    RO_TRY(ensure(c, c->x_mb, (n_parents + 1) * sizeof(uint32_t), "member bases"));
    RO_TRY(ensure(c, c->x_coff, std::max<uint64_t>(n_parents, 1) * sizeof(uint32_t), "member bases"));
    RO_TRY(ensure(c, c->x_mtfp, mtfp_cap * sizeof(uint32_t), "member tiles"));
    RO_TRY(ensure(c, c->x_hdr, sizeof(ListHdr), "list header"));
    aa.list.parents = d_parents;
    aa.list.status = d_status;
    aa.list.mb = (uint32_t*)c->x_mb.p;
    aa.list.coff = (uint32_t*)c->x_coff.p;
    aa.list.mtfp = (uint32_t*)c->x_mtfp.p;
    aa.list.mtfp_cap = mtfp_cap;
    aa.list.hdr = (ListHdr*)c->x_hdr.p;
    RO_TRY(tile_status(c, TS_ASM_PARENTS, ceil_div(n_parents, (uint64_t)AP_THREADS * AP_ITEMS),
                       &aa.ts_parents));
  } else {
    LS = &S.lists[x->last_list];
    aa.list = list_bufs(*LS, mtfp_cap);
  }
  if (!planned) {
    RO_TRY(tile_status(c, TS_ASM_MEMBERS, ceil_div(member_cap, (uint64_t)AM_TILE), &aa.ts_members));

    // planning follows everything enqueued on the context's stream so far,
    // and the copy that last read this plan slot
    RO_TRY(order(c, c->fork, c->stream, c->plan_stream));
    RO_TRY(order(c, c->fin_plan, c->fin_stream[c->last_fin], c->plan_stream));   // the commit's list
    RO_TRY(ev_wait(c, PS.freed, c->plan_stream));
    if (c->plan_stream != c->copy_stream) {
      // caller memory planning writes (list structure; a caller's list's
      // outcomes) against what copies still in flight write
      ro_ctx::Span pw[5];
      int npw = 0;
      auto span = [](const void* p, uint64_t bytes) {
        return ro_ctx::Span{(uintptr_t)p, (uintptr_t)p + (uintptr_t)bytes};
      };
      if (d_parents) pw[npw++] = span(d_status, n_parents);
      if (eo) {
        pw[npw++] = span(eo->base, (n_parents + 1) * sizeof(uint64_t));
        pw[npw++] = span(eo->state, eo->cap);
        pw[npw++] = span(eo->off, eo->cap * sizeof(uint64_t));
        pw[npw++] = span(eo->len, eo->cap * sizeof(uint32_t));
      }
      bool meet = npw > 0 && c->copy_spans_full;
      for (int i = 0; i < npw && !meet; ++i)
        for (const auto& b : c->copy_spans)
          if (pw[i].lo < pw[i].hi && pw[i].lo < b.hi && b.lo < pw[i].hi) {
            meet = true;
            break;
          }
      if (meet) RO_TRY(ev_wait(c, c->copy_done, c->plan_stream));
    }
    launch_assemble_plan(c->Lp, aa);
    RO_TRY(check_launch(c, "assemble (plan)"));
    if (!LS && c->plan_stream != c->stream) {
      // a caller's list is classified against the parents' counters as they
      // are now: later commits wait for that
      RO_TRY(order(c, c->x_planned, c->plan_stream, c->stream));
    }
    RO_TRY(order(c, PS.ready, c->plan_stream, c->copy_stream));
  }
  launch_assemble_copy(c->Lc, aa);
  RO_TRY(check_launch(c, "assemble (copy)"));
  if (c->copy_stream != c->plan_stream) {
    if (!planned) RO_TRY(ev_record(c, PS.freed, c->copy_stream));
    RO_TRY(ev_record(c, c->copy_done, c->copy_stream));
    // what this copy writes of the caller's memory (the bytes of d_out are
    // written by copies only)
    auto add = [&](const void* p, uint64_t bytes) {
      if (!p || !bytes) return;
      if (c->copy_spans.size() >= ro_ctx::MAX_SPANS) {
        c->copy_spans_full = true;
        return;
      }
      c->copy_spans.push_back({(uintptr_t)p, (uintptr_t)p + (uintptr_t)bytes});
    };
    if (!d_parents) add(d_status, n_parents);
    add(d_out_off, (n_parents + 1) * sizeof(uint64_t));
    add(d_out_len, n_parents * sizeof(uint32_t));
    if (eo) add(eo->off, eo->cap * sizeof(uint64_t));
  }
  // the copy reads the list's outcomes: the slot is free once it is done
  if (LS && c->copy_stream != c->stream) RO_TRY(ev_record(c, LS->freed, c->copy_stream));
  x->assembles += 1;
  if (h_out_bytes || (eo && eo->h_n)) {
    ro_status st = sync_and_check(c);
    if (h_out_bytes) *h_out_bytes = c->hs->as_bytes;
    if (eo && eo->h_n) *eo->h_n = c->hs->as_elems;
    return st;
  }
  return RO_OK;
}
}  // namespace
