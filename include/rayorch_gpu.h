/*
 * rayorch_gpu.h — C ABI of the GB300 (sm_103a) lineage expand / gather path.
 *
 * The library keeps, on one GPU, the structural lineage state that RayOrch
 * (arXiv 2609.18703) maintains for an ordered, variable-cardinality
 * parent -> child expansion and its matching ordered gather:
 *
 *   ro_expand         Section 4.2, Table 2, Eq. (1): child offsets, each
 *                     child's immediate parent and immutable ordinal.
 *   ro_batch_ready    Section 4.3, Eq. (2): per-Call FIFO Ready Queue and
 *                     elastic reservation into fixed-size batches.
 *   ro_batch_ready_parent  Section 4.3: the same queue with parent-bound
 *                     reservation (each batch holds siblings of one parent).
 *   ro_gather_commit  Section 4.4, Eq. (3) and Section 4.2 (Reduce):
 *                     generation-fenced commit of out-of-order child results,
 *                     per-parent terminal counting, completed-parent list.
 *   ro_assemble       Section 4.2 (Reduce): each completed parent's Present
 *                     child payloads concatenated in ordinal order.
 *
 * Conventions for every entry point
 * ---------------------------------
 * - Pointers prefixed d_ are device memory of the context's GPU; h_ are host
 *   memory.  The caller allocates and owns every pointer it passes; the
 *   library never keeps a caller pointer beyond the call (except the arena,
 *   see ro_gather_commit).  A context owns its internal lineage state
 *   (phase words, result slots, parent counters, queues, scratch).
 * - Work is issued on the context's stream, in call order, except assembly,
 *   completion lists and admissions: ro_assemble plans on the context's plan
 *   stream and copies on its copy stream, with separate streams set
 *   (ro_ctx_set_streams) ro_gather_commit builds its completed-parent list
 *   and that list's copy plan on one of three streams the context owns
 *   (commits take them in turn), and with Call streams set
 *   (ro_ctx_set_call_streams) ro_batch_ready runs on its Call's stream.
 *   Each assembly is ordered after all work the caller issued on the
 *   context before it; the caller's ro_assemble
 *   outputs and ro_gather_commit's d_done_parents / d_n_done are complete
 *   once ro_ctx_join has made the context's stream wait for the others (or
 *   once any call synchronises).  Calls return without waiting for the
 *   GPU unless an h_ output is requested: a non-NULL h_ pointer makes the
 *   call synchronise every stream and fill it in.  The d_ count outputs are
 *   written by the GPU in stream order, so a following call can consume
 *   them (the d_n inputs) without a host round trip.
 * - Errors are returned as ro_status; nothing throws across the ABI.
 *   Argument errors the host can see are RO_E_INVAL with no side effects.
 *   Conditions only the GPU can see (an output too small, a wait that timed
 *   out) are recorded in the context and returned by the next call that
 *   synchronises (any call with an h_ output, or ro_ctx_sync); the call that
 *   hit them leaves lineage state as it was.  CUDA runtime errors give
 *   RO_E_CUDA and stick to the context.
 * - Limits: fewer than 2^32 parents and 2^32 children per expansion; arena
 *   offsets and sizes below 2^48; at most 256 Calls per context; payload
 *   lengths are uint32.
 */
#ifndef RAYORCH_GPU_H
#define RAYORCH_GPU_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct ro_ctx ro_ctx;
typedef int32_t ro_status;

/* call status */
enum {
  RO_OK = 0,
  RO_E_INVAL = 1,     /* bad argument; nothing changed */
  RO_E_CAPACITY = 2,  /* an output buffer is too small; nothing changed, retry */
  RO_E_OVERFLOW = 3,  /* a count or size exceeds the limits above */
  RO_E_STATE = 4,     /* the call does not fit the lineage state (unknown xid, ...) */
  RO_E_OOM = 5,       /* device memory for internal state could not be allocated */
  RO_E_CUDA = 6,      /* a CUDA runtime error; sticky until ro_ctx_destroy */
  RO_E_TIMEOUT = 7    /* a bounded device-side wait gave up; results of that call are void */
};

/* Item outcomes of Eq. (1), as carried by reports and by assembled parents */
enum {
  RO_PENDING = 0,     /* not (yet) complete */
  RO_PRESENT = 1,
  RO_DROPPED = 2,
  RO_FAILED = 3,
  RO_SUPPRESSED = 4
};
/* A report kind that is not an outcome (Section 4.4, typed GroupFailure):
 * the reporting Grain failed (it is sealed RO_FAILED) and a barrier is
 * installed for its (Call, parent): every sibling not yet sealed is sealed
 * RO_SUPPRESSED at once.  Queued siblings then leave the Ready Queue at the
 * next reservation without being dispatched, later reports of in-flight
 * siblings are rejected (RO_REJ_BARRIER), siblings sealed earlier keep their
 * facts and other parents are unaffected. */
enum { RO_GROUP_FAILURE = 5 };

/* per-report verdict of the generation fence, Eq. (3) */
enum {
  RO_ACCEPT = 0,
  RO_REJ_INVALID = 1,       /* no such child, unknown outcome, or payload outside the arena */
  RO_REJ_NOT_INFLIGHT = 2,  /* the child's Grain is WAITING or READY */
  RO_REJ_STALE_GEN = 3,     /* generation differs from the Grain's current one */
  RO_REJ_DUPLICATE = 4,     /* the Grain is already SEALED (earlier report, or an earlier
                               report of the same call) */
  RO_REJ_BARRIER = 5        /* the Grain was sealed by a sibling's GroupFailure */
};

/* cumulative counters of a context (since create or the last reset) */
typedef struct {
  uint64_t accepted, rej_invalid, rej_not_inflight, rej_stale_gen, rej_duplicate;
  uint64_t ready_bad_candidates;  /* batch_ready candidates naming no child */
  uint64_t assemble_incomplete;   /* assembled list entries that were not complete */
  uint64_t rej_barrier;           /* reports rejected with RO_REJ_BARRIER */
  uint64_t barrier_not_dispatched;/* siblings a GroupFailure sealed while WAITING or READY */
  uint64_t barrier_in_flight;     /* siblings a GroupFailure sealed while IN-FLIGHT */
  uint64_t queue_dropped;         /* sealed Grains removed from a Ready Queue undispatched */
  uint64_t retried;               /* Grains ro_retry moved back to READY */
  uint64_t retry_skipped;         /* ro_retry entries naming no IN-FLIGHT Grain of the Call */
} ro_stats;

/* ------------------------------------------------------------------------
 * Context = one source microbatch (Sections 1 and 4.3: Ready Queues and
 * ordered gathering are scoped to one input microbatch).  `stream` is a
 * cudaStream_t (NULL = legacy default stream) on device `device`; n_calls in
 * [1, 256] is the number of Calls whose Ready Queues the context keeps.
 * Two environment variables, read here, tune the context: RO_COPY_SMALL_CHUNKS
 * (copies of at most this many 16 KB chunks take the direct path; default
 * 256, 0 stages every copy) and RO_ADMIT_TWO_PASS (non-zero: every
 * admission takes the two-pass path instead of the one-pass cooperative
 * kernel that lists of up to a few thousand tiles of 2,048 candidates use).
 */
ro_status ro_ctx_create(ro_ctx** ctx, int32_t device, void* stream, uint32_t n_calls);
ro_status ro_ctx_destroy(ro_ctx* ctx);
/* Forget every expansion (start the next microbatch).  Device memory is kept
 * and reused by later expansions of the same or smaller size. */
ro_status ro_ctx_reset(ro_ctx* ctx);
/* Wait for every stream of the context and return (then clear) any condition
 * recorded by the GPU. */
ro_status ro_ctx_sync(ro_ctx* ctx);
/* Streams for assembly (no counterpart in the paper; it schedules the path).
 * plan_stream and copy_stream are cudaStream_t handles on the context's
 * device, NULL for the context's stream.  With separate streams the planning
 * and copy of one wave's completed parents overlap the next waves' admission
 * and commits; up to four commits and assemblies per expansion may be in
 * flight at once (the context keeps four list and plan slots per expansion
 * and orders their reuse with events).  With a plan stream other than the
 * context's stream, the context also creates three streams of its own
 * (destroyed with the context) for the commits' completed-parent lists and
 * their copy plans, which consecutive commits take in turn: one commit's
 * list is built while the next commits' reports are applied and the next
 * two commits' lists are built (32 completion bitmaps per expansion, taken
 * in turn).  The context's stream first waits for the old streams.  The caller keeps the streams alive until ro_ctx_destroy
 * or the next ro_ctx_set_streams. */
ro_status ro_ctx_set_streams(ro_ctx* ctx, void* plan_stream, void* copy_stream);
/* Streams for the Calls' admissions (Section 4.3: each Call has its own
 * Ready Queue, and the queues are independent).  streams[k] (a cudaStream_t
 * on the context's device, or NULL for the context's stream) runs
 * ro_batch_ready for Call k, k < n; Calls from n on use the context's
 * stream.  An admission on a Call's stream follows everything issued on
 * the context's stream before it, so the admissions of several Calls
 * issued one after another run at the same time; the context's stream
 * waits for them before its next launch (any other call that works on the
 * expansion: ro_expand, ro_gather_commit, ro_retry, ro_batch_ready_parent,
 * ro_assemble) and in ro_ctx_join.  Each Call's outputs (d_batched,
 * d_n_batched) are written on its stream: give Calls that run at the same
 * time outputs of their own.  ro_batch_ready_parent always runs on the
 * context's stream.  The context's stream first waits for the old streams;
 * the caller keeps the streams alive until ro_ctx_destroy or the next call
 * of this function.
 * Errors: RO_E_INVAL if n exceeds the context's Calls or streams is NULL
 * with n > 0. */
ro_status ro_ctx_set_call_streams(ro_ctx* ctx, void* const* streams, uint32_t n);
/* Make the context's stream wait (on the GPU) for all work issued so far on
 * the plan and copy streams, the context's three completion streams and the
 * Calls' streams.  Call it before reading assembly outputs in
 * stream order, before starting a capture of the context's stream, and
 * before ending one (a captured assembly forks onto the other streams, and a
 * capture must join them back).  Nothing waits on the host. */
ro_status ro_ctx_join(ro_ctx* ctx);
/* Self-test of the bounded device-side waits.  Every wait of the lineage
 * kernels gives up after a bounded number of polls (about two seconds),
 * records the time-out in the context and returns, so that a wait that can
 * never end (a lost dependency) turns into RO_E_TIMEOUT instead of a hung
 * GPU.  This call runs one such wait that nothing releases, on scratch state
 * of its own: kind 0 a decoupled look-back whose predecessor tile never
 * publishes, kind 1 a grid barrier of two CTAs one of which never arrives.
 * It synchronises and returns RO_E_TIMEOUT when the wait gave up and was
 * reported (the expected outcome), RO_OK if it was not (a defect).  Lineage
 * state is untouched; the context stays usable.
 * Errors: RO_E_INVAL for another kind; an earlier call's pending device
 * error is returned first. */
ro_status ro_ctx_selftest_timeout(ro_ctx* ctx, uint32_t kind);
/* Synchronise and copy the cumulative counters. */
ro_status ro_ctx_stats(ro_ctx* ctx, ro_stats* out);
/* Text of the last error on this context ("" if none).  Valid until the next call. */
const char* ro_last_error(const ro_ctx* ctx);

/* Kernel ids for the profiling calls below, in launch order of the path. */
enum {
  RO_K_EXPAND_SCAN = 0, RO_K_EXPAND_FILL = 1, RO_K_READY_COUNT = 2, RO_K_READY_SCATTER = 3,
  RO_K_COMMIT_SCATTER = 4, RO_K_COMMIT_PLAN = 5, RO_K_ASM_PARENTS = 6, RO_K_ASM_MEMBERS = 7,
  RO_K_ASM_COPY = 8, RO_K_RETRY_CLAIM = 9, RO_K_RETRY_SCATTER = 10, RO_K_PB_KEYS = 11,
  RO_K_PB_HIST = 12, RO_K_PB_ROWSCAN = 13, RO_K_PB_SORT = 14, RO_K_PB_BOUNDS = 15,
  RO_K_PB_HEADS = 16, RO_K_PB_MARK = 17, RO_K_PB_SCAN = 18, RO_K_PB_EMIT = 19,
  RO_K_COMMIT_FIX = 20, RO_K_READY_FUSED = 21, RO_K_COUNT = 22
};
/* Tracing (no counterpart in the paper; it instruments the path).  Every
 * kernel launch is counted; kernels whose bit (1 << RO_K_*) is set in
 * kernel_mask are also bracketed by a pair of CUDA events on the context's
 * stream.  Recording events costs host time per launch, so time few kernels. */
ro_status ro_ctx_profile(ro_ctx* ctx, uint32_t kernel_mask);
/* Synchronise, then copy per kernel (arrays of n_kernels entries, any may be
 * NULL): launches since the last read, launches timed, and their summed
 * device milliseconds.  Resets the counters. */
ro_status ro_ctx_profile_read(ro_ctx* ctx, uint64_t* launches, uint64_t* timed, double* ms,
                              uint32_t n_kernels);

/* ------------------------------------------------------------------------
 * ro_expand — materialise one Expansion (Section 4.2; Table 2 gives the child
 * key (parent, ordinal); Eq. (1) makes an empty child list terminal).
 *
 *   parent_xid    -1 for a root expansion, else the xid whose children are
 *                 the parents here (nested levels); n_parents must then equal
 *                 that expansion's child count.
 *   d_counts      uint32[n_parents]  children of each parent (read only).
 *   d_parent_call uint8[n_parents] or NULL: the Call that consumes each
 *                 parent's children (NULL: Call 0).
 *   d_offsets     uint64[n_parents+1] out: exclusive prefix sum of counts;
 *                 d_offsets[n_parents] = number of children N.
 *   d_child_parent, d_child_ordinal  uint32[child_cap] out: for child c
 *                 (numbered parent-major, c = d_offsets[p] + ordinal) its
 *                 immediate parent and zero-based ordinal.
 *   d_empty_parents uint32[n_parents] out or NULL: ascending ids of parents
 *                 with no children; they are complete at once and can be
 *                 assembled (Present, empty).
 *   h_n_children, h_n_empty  out (required / optional): N and the number
 *                 of empty parents.  This call always synchronises.
 *   xid           out: handle of the new expansion.
 * Errors: RO_E_CAPACITY if N > child_cap (h_n_children holds N, no expansion
 * is created); RO_E_OVERFLOW if N >= 2^32.
 */
ro_status ro_expand(ro_ctx* ctx, int32_t parent_xid, const uint32_t* d_counts,
                    uint64_t n_parents, const uint8_t* d_parent_call, uint64_t* d_offsets,
                    uint32_t* d_child_parent, uint32_t* d_child_ordinal, uint64_t child_cap,
                    uint32_t* d_empty_parents, uint64_t* h_n_children, uint64_t* h_n_empty,
                    int32_t* xid);

/* ------------------------------------------------------------------------
 * ro_batch_ready — admission into the per-Call FIFO Ready Queue and elastic
 * reservation (Section 4.3, Eq. 2).
 *
 * Candidates are taken in order; a candidate enters Call `call`'s queue of
 * expansion xid (WAITING -> READY) when it names a child of xid whose Grain
 * is WAITING and which belongs to that Call.  A child named twice enters once,
 * at its first position.  Then whole batches of batch_size are taken from the
 * head of the queue (READY -> IN-FLIGHT); with flush != 0 the trailing partial
 * batch is taken too.  Entries left in the queue stay READY for the next call.
 *
 *   d_cand      uint32[n_cand] child ids in readiness order, or NULL for all
 *               children of xid in id order (n_cand ignored).  n_cand < 2^30.
 *   d_batched   uint32[batched_cap] out: the reserved children; batch k is
 *               d_batched[k*batch_size ...].  Batches mix parents freely.
 *   d_n_batched uint64 out (device) or NULL: number reserved.
 *   h_n_batched, h_n_batches out (host) or NULL: number reserved and number of
 *               batches; either makes the call synchronise.
 * Errors: RO_E_CAPACITY when more would be reserved than batched_cap (reported
 * when the context next synchronises; queue and phases unchanged).
 */
ro_status ro_batch_ready(ro_ctx* ctx, int32_t xid, uint32_t call, const uint32_t* d_cand,
                         uint64_t n_cand, uint32_t batch_size, int32_t flush,
                         uint32_t* d_batched, uint64_t batched_cap, uint64_t* d_n_batched,
                         uint64_t* h_n_batched, uint64_t* h_n_batches);

/* ------------------------------------------------------------------------
 * ro_batch_ready_calls — the admissions of n Calls from one candidate list
 * (Section 4.3: each Call keeps a Ready Queue of its own), in one launch.
 *
 * The result equals ro_batch_ready(ctx, xid, calls[k], d_cand, n_cand,
 * batch_size, flush, d_batched[k], batched_cap[k], d_n_batched[k], NULL,
 * NULL) for k = 0 .. n-1 in turn (each Call admits only its own children,
 * into its own queue, so the Calls' admissions are independent).  Runs on
 * the context's stream, after the Calls' pending admissions on their own
 * streams: one cooperative kernel over all n Calls when the list's tiles fit
 * the device at once (n times (n_cand / 2048 + 1) CTAs), else one admission
 * after another.
 *
 *   calls        host uint32[n]: distinct Calls, n in [1, 8].
 *   d_batched    host array of n device pointers (uint32[batched_cap[k]] out).
 *   batched_cap  host uint64[n].
 *   d_n_batched  host array of n device pointers (uint64 out, each may be
 *                NULL), or NULL.
 * Errors: RO_E_INVAL (n out of range, a Call named twice or out of range,
 * NULL arrays) with no side effects; a reservation larger than a Call's
 * capacity refuses that Call's admission only (RO_E_CAPACITY at the next
 * synchronising call; that Call's queue and phases unchanged).
 */
ro_status ro_batch_ready_calls(ro_ctx* ctx, int32_t xid, uint32_t n, const uint32_t* calls,
                               const uint32_t* d_cand, uint64_t n_cand, uint32_t batch_size,
                               int32_t flush, uint32_t* const* d_batched,
                               const uint64_t* batched_cap, uint64_t* const* d_n_batched);

/* ------------------------------------------------------------------------
 * ro_batch_ready_parent — admission into the per-Call FIFO Ready Queue and
 * parent-bound reservation (Section 4.3, Eq. 2).
 *
 * Admission is that of ro_batch_ready.  Then reservations are made one after
 * another: each takes up to batch_size queued siblings of the parent of the
 * queue's first entry, in queue order (READY -> IN-FLIGHT), and every entry
 * it leaves keeps its place relative to the others.  Without flush a
 * reservation that would hold fewer than batch_size siblings is not made and
 * the queue waits for more of that parent's siblings (as ro_batch_ready waits
 * for a whole batch); with flush != 0 reservations repeat until the queue is
 * empty.  Recovery groups (ro_retry) enter ahead of the queue's entries first.
 *
 *   d_cand, n_cand, batch_size, flush   as in ro_batch_ready.
 *   d_batched    uint32[batched_cap] out: the batches back to back; each
 *                holds children of one parent.
 *   d_batch_off  uint64[batch_off_cap] out or NULL: n_batches + 1 batch
 *                boundaries; batch k is d_batched[d_batch_off[k] ..
 *                d_batch_off[k+1]).
 *   d_n_batched, d_n_batches  uint64 out (device) or NULL.
 *   h_n_batched, h_n_batches  out (host) or NULL; either makes the call
 *                synchronise.
 * Errors: RO_E_CAPACITY when more would be reserved than batched_cap, or
 * d_batch_off cannot hold n_batches + 1 entries (reported when the context
 * next synchronises; the admission is undone, the outputs are undefined).
 * Device scratch of about 37 bytes per child and 8 per parent of the
 * expansion is allocated at the first call (like ro_batch_ready, this call
 * cannot be the first to size it inside a stream capture).
 */
ro_status ro_batch_ready_parent(ro_ctx* ctx, int32_t xid, uint32_t call, const uint32_t* d_cand,
                                uint64_t n_cand, uint32_t batch_size, int32_t flush,
                                uint32_t* d_batched, uint64_t batched_cap, uint64_t* d_batch_off,
                                uint64_t batch_off_cap, uint64_t* d_n_batched,
                                uint64_t* d_n_batches, uint64_t* h_n_batched,
                                uint64_t* h_n_batches);

/* ------------------------------------------------------------------------
 * ro_retry — a failed physical attempt is tried again (Section 4.4: the
 * runtime may retry a Grain at a higher generation; Eq. 2's IN-FLIGHT ->
 * READY edge; Section 4.3: recovery queues reinsert the Grain group).
 *
 *   d_children  uint32[n] the Grains of the failed attempt (a batch), in
 *               the order they are to run again.
 * Every listed Grain of Call `call` that is IN-FLIGHT (first occurrence in
 * the list) goes back to READY with its generation + 1, so reports of the
 * failed attempt are rejected (RO_REJ_NOT_INFLIGHT while READY,
 * RO_REJ_STALE_GEN once dispatched again).  Those Grains, in list order,
 * form one group of the Call's recovery queue; the next ro_batch_ready for
 * the Call reserves recovery groups, oldest first, before the Ready Queue's
 * entries (a retried Grain that a GroupFailure has sealed meanwhile is
 * dropped).  Entries naming no IN-FLIGHT Grain of the Call are skipped and
 * counted.  h_n_retried (host, synchronises) out or NULL: Grains retried.
 */
ro_status ro_retry(ro_ctx* ctx, int32_t xid, uint32_t call, const uint32_t* d_children, uint64_t n,
                   uint64_t* h_n_retried);

/* ------------------------------------------------------------------------
 * ro_gather_commit — generation-fenced commit of child results (Section 4.4,
 * Eq. 3) and per-parent completion (Section 4.2, Reduce).
 *
 * Report r names child d_child[r] with outcome d_state[r] (RO_PRESENT,
 * RO_DROPPED, RO_FAILED or RO_SUPPRESSED) or the kind RO_GROUP_FAILURE
 * (Section 4.4, see above); a Present report's value is the
 * d_len[r] bytes at arena offset d_arena_off[r] (ignored for other outcomes).
 * A report is accepted when the child's Grain is IN-FLIGHT and d_gen[r] is
 * its current generation; the Grain becomes SEALED and the outcome is
 * published for good.  Reports of one call are applied as if one after
 * another in array order (the first of several reports for one Grain wins;
 * a GroupFailure's barrier applies to the reports after it, not before).
 * A parent completes when all of its children are sealed.
 *
 *   n, d_n      report count (host), or a device uint64 count (d_n != NULL;
 *               n is then an upper bound used for launch sizing).
 *   d_gen       uint32[n] or NULL (generation 0).
 *   arena_bytes size of the result arena the offsets refer to.  The arena
 *               bytes of accepted Present reports must stay unchanged until
 *               their parents are assembled.
 *   d_code      uint8[n] out or NULL: RO_ACCEPT or an RO_REJ_* verdict.
 *               Rejected reports change nothing.
 *   d_done_parents uint32[done_cap] out or NULL: parents completed by this
 *               call, ascending.  done_cap must be >= min(n, parents of xid).
 *   d_n_done (device) / h_n_done (host, synchronises) out or NULL.
 *   With separate streams set, d_done_parents and d_n_done are written on
 *   one of the context's completion streams (see the conventions above);
 *   ro_assemble orders itself after them.  The same pass plans the copy of
 *   the completed parents, so ro_assemble of this list (d_parents NULL,
 *   without list structure) runs only the copy.
 * Capture: a captured commit keeps the context's commit number it was
 * captured with; replay a captured sequence of commits on a fresh expansion
 * (ro_expand clears the GroupFailure barrier table), as a new microbatch.
 */
ro_status ro_gather_commit(ro_ctx* ctx, int32_t xid, uint64_t n, const uint64_t* d_n,
                           const uint32_t* d_child, const uint8_t* d_state,
                           const uint32_t* d_len, const uint64_t* d_arena_off,
                           const uint32_t* d_gen, uint64_t arena_bytes, uint8_t* d_code,
                           uint32_t* d_done_parents, uint64_t done_cap, uint64_t* d_n_done,
                           uint64_t* h_n_done);

/* ------------------------------------------------------------------------
 * ro_assemble — ordered Reduce output (Section 4.2).
 *
 * For each listed parent: if it is not complete, status RO_PENDING and no
 * bytes; if a child Failed or was Suppressed, RO_SUPPRESSED and no bytes;
 * otherwise RO_PRESENT and the Present children's payloads concatenated in
 * ordinal order (Dropped children add nothing; no survivors give 0 bytes).
 * Parents are written back to back, in list order, starting at d_out + base
 * where base = *d_out_cursor (if given) or 0; the cursor then advances.
 *
 *   d_arena      the result arena the committed reports referred to.  It
 *                is read in aligned 16-byte blocks, so the memory from
 *                d_arena up to the next 16-byte boundary at or after
 *                d_arena + arena_bytes must be readable (true of any
 *                cudaMalloc allocation that holds the arena).  The arena
 *                may be pinned host memory (cudaHostAlloc / cudaHostRegister):
 *                the copy then reads the needed payload bytes in place over
 *                the host link with plain loads (no staging copy of the
 *                arena).  Pageable host memory is refused (RO_E_INVAL).
 *   d_parents    uint32[n_parents] parent ids, or NULL for the parents
 *                completed by the latest ro_gather_commit on xid (in its
 *                ascending order); n_parents is then the capacity of the
 *                per-parent outputs.  d_n_parents (device count) may replace
 *                n_parents for an explicit list.
 *   d_status     uint8[n] out; d_out_off uint64[n+1] out: byte offsets into
 *                d_out (entry n = end); d_out_len uint32[n] out or NULL.
 *                With d_out_len, RO_E_OVERFLOW if a parent exceeds 2^32-1 bytes.
 *   d_out        uint8[out_cap] out.  Byte-exact, no padding; any alignment.
 *                May be pinned host memory (written in place by the copy).
 *   d_out_bytes (device) / h_out_bytes (host, synchronises) out or NULL:
 *                bytes written by this call.
 * Together, (d_parents or the commit's list, d_status, d_out_len, d_out_off)
 * have the layout of a report array, so an assembled level can be committed
 * as the results of the level above (nested expansions).
 * Errors: RO_E_CAPACITY when base + bytes > out_cap or the list is longer
 * than n_parents (nothing is copied).
 * Streams: the latest commit's list (d_parents NULL) was planned by the
 * commit, so only the copy runs, on the copy stream; an explicit list is
 * planned on the plan stream first (see ro_ctx_set_streams).  The outputs
 * (d_status, d_out_off, d_out_len, d_out, the cursor, d_out_bytes) are
 * written by the copy.  A d_arena smaller than the accepted reports'
 * ranges is refused on the GPU (RO_E_INVAL, nothing copied).  Read them after
 * ro_ctx_join in stream order, or after any synchronising call.
 * Consecutive calls may pass the same output arrays: their writes land in
 * call order (a call whose planning writes caller memory that an earlier
 * call's copy is still writing waits for that copy).
 */
ro_status ro_assemble(ro_ctx* ctx, int32_t xid, const uint8_t* d_arena, uint64_t arena_bytes,
                      const uint32_t* d_parents, uint64_t n_parents, const uint64_t* d_n_parents,
                      uint8_t* d_status, uint64_t* d_out_off, uint32_t* d_out_len,
                      uint8_t* d_out, uint64_t out_cap, uint64_t* d_out_cursor,
                      uint64_t* d_out_bytes, uint64_t* h_out_bytes);

/* ------------------------------------------------------------------------
 * ro_assemble_list — ro_assemble plus the list structure of each assembled
 * parent (Section 4.2: the Reduce emits the present values in immutable
 * ordinal order; Table 3's F.reduce gathers a list), so a reader can split
 * each parent's concatenated bytes back into its ordered list.
 *
 * All arguments of ro_assemble, then:
 *   d_elem_base  uint64[n+1] out: listed parent i's entries are
 *                d_elem_base[i] .. d_elem_base[i+1]-1 (none unless it is
 *                assembled Present).
 *   d_elem_state uint8[elem_cap] out: per entry, in ordinal order, the
 *                member's outcome (RO_PRESENT or RO_DROPPED).
 *   d_elem_off   uint64[elem_cap] out: the offset in d_out of the member's
 *                bytes (a Dropped member: where it would have been).
 *   d_elem_len   uint32[elem_cap] out: the member's bytes (0 if Dropped).
 *   elem_cap     entries the three arrays hold: every member of every listed
 *                Present parent is an entry.
 *   d_n_elems (device) / h_n_elems (host, synchronises) out or NULL: entries.
 * Errors: those of ro_assemble; RO_E_CAPACITY also when the entries exceed
 * elem_cap (then nothing is copied and the entry arrays are undefined).
 * A parent whose members were all Dropped is Present with 0 bytes and its
 * entries all RO_DROPPED: a present empty list.
 */
ro_status ro_assemble_list(ro_ctx* ctx, int32_t xid, const uint8_t* d_arena, uint64_t arena_bytes,
                           const uint32_t* d_parents, uint64_t n_parents,
                           const uint64_t* d_n_parents, uint8_t* d_status, uint64_t* d_out_off,
                           uint32_t* d_out_len, uint8_t* d_out, uint64_t out_cap,
                           uint64_t* d_out_cursor, uint64_t* d_out_bytes, uint64_t* h_out_bytes,
                           uint64_t* d_elem_base, uint8_t* d_elem_state, uint64_t* d_elem_off,
                           uint32_t* d_elem_len, uint64_t elem_cap, uint64_t* d_n_elems,
                           uint64_t* h_n_elems);

/* ------------------------------------------------------------------------
 * ro_filter_reports — F.filter (Table 3: pass on true, drop on false) on a
 * batch of reports before they are committed, with Section 4.2's
 * propagation precedence: a RO_PRESENT report whose d_keep byte is 0
 * becomes RO_DROPPED; every other report keeps its state (a failed or
 * suppressed input stays so).  d_state uint8[n] in/out, d_keep uint8[n];
 * runs on the context's stream.
 */
ro_status ro_filter_reports(ro_ctx* ctx, uint8_t* d_state, const uint8_t* d_keep, uint64_t n);

/* ------------------------------------------------------------------------
 * ro_expand_noalloc — the offsets, parents and ordinals of ro_expand, for
 * callers that cannot allocate device memory.  The paper has no counterpart;
 * this is a deployment variant.
 *
 * Some callers cannot call cudaMalloc: code that runs inside a memory budget
 * owned by another allocator, code that must not synchronise the device the
 * way cudaMalloc/cudaFree may, or embedders that forbid allocation after
 * start-up.  This call needs no context and allocates nothing.  Its scratch
 * (scan tile status, fill-tile table, counters) is one fixed array of about
 * 292 KB in the library's device memory, which every GPU that loads the
 * library holds until the process exits.  It keeps no lineage state, so the
 * result cannot be committed or assembled against.
 *
 *   Arguments as in ro_expand (d_counts, n_parents, d_offsets uint64[P+1],
 *   d_child_parent / d_child_ordinal uint32[child_cap], d_empty_parents
 *   uint32[P] or NULL), on `stream` (a cudaStream_t, NULL = legacy default
 *   stream) of the current device.  h_n_children (required) and h_n_empty
 *   (optional) receive N and the number of empty parents.  The call
 *   returns only after all of its work on `stream` has finished (it
 *   synchronises the stream after the scan and again after the fill), so
 *   its outputs are complete on return and the scratch is free for the
 *   next call.
 *   Limits: at most 16,777,216 parents and 134,217,728 children, else
 *   RO_E_CAPACITY (beyond the static scratch; nothing is launched when the
 *   parent count is too large).  RO_E_CAPACITY also when N > child_cap.
 *   When the children are refused (too many for the scratch or for
 *   child_cap) the scan has run: d_offsets, d_empty_parents and the counts
 *   are written, the child arrays are not, and the next call is unaffected.
 *   The first call on a device looks up the scratch's device address; make
 *   that first call before any stream capture.  All calls share the one
 *   scratch array: calls that overlap on the GPU (other streams, other host
 *   threads) race and must be serialised by the caller.
 */
ro_status ro_expand_noalloc(const uint32_t* d_counts, uint64_t n_parents, uint64_t* d_offsets,
                            uint32_t* d_child_parent, uint32_t* d_child_ordinal,
                            uint64_t child_cap, uint32_t* d_empty_parents, void* stream,
                            uint64_t* h_n_children, uint64_t* h_n_empty);

#ifdef __cplusplus
}
#endif
#endif /* RAYORCH_GPU_H */
