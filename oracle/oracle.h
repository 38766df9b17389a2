/*
 * oracle.h — plain, single-threaded CPU statement of the lineage expand /
 * ready-queue batch / gather-commit / assemble semantics of RayOrch
 * (arXiv 2609.18703, Sections 4.2-4.5).
 *
 * TEST INFRASTRUCTURE ONLY.  Only the test suite, the smoke check and the
 * benchmark's CPU-baseline leg may load or call this code.  It shares no
 * code, header, table or helper with the GPU library; both follow the paper.
 *
 * Every array is host memory.  Sizes are element counts.  Status and code
 * numbering is the same as the GPU library's so that outputs compare
 * directly; the numbers are restated here, not included from there.
 */
#ifndef RO_ORACLE_H
#define RO_ORACLE_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* call status */
enum { OR_OK = 0, OR_E_INVAL = 1, OR_E_CAPACITY = 2, OR_E_OVERFLOW = 3, OR_E_STATE = 4,
       OR_E_OOM = 5 };
/* Item outcomes of Eq. (1) as carried by reports and assembled parents */
enum { OR_PENDING = 0, OR_PRESENT = 1, OR_DROPPED = 2, OR_FAILED = 3, OR_SUPPRESSED = 4 };
/* A report kind, not an outcome (Section 4.4, typed GroupFailure): the
 * reporting Grain Failed and its siblings under the same (Call, parent)
 * are to be suppressed. */
enum { OR_GROUP_FAILURE = 5 };
/* per-report verdicts of the generation fence, Eq. (3); BARRIER: the Grain
 * was sealed by a GroupFailure of a sibling */
enum { OR_ACCEPT = 0, OR_REJ_INVALID = 1, OR_REJ_NOT_INFLIGHT = 2, OR_REJ_STALE_GEN = 3,
       OR_REJ_DUPLICATE = 4, OR_REJ_BARRIER = 5 };
/* Grain phases of Eq. (2) */
enum { OR_WAITING = 0, OR_READY = 1, OR_IN_FLIGHT = 2, OR_SEALED = 3 };

typedef struct or_ctx or_ctx;

typedef struct {
  uint64_t accepted, rej_invalid, rej_not_inflight, rej_stale_gen, rej_duplicate;
  uint64_t ready_bad_candidates;    /* candidates naming no child of the expansion */
  uint64_t assemble_incomplete;     /* listed parents that were not complete */
  uint64_t rej_barrier;             /* reports for Grains a GroupFailure suppressed */
  uint64_t barrier_not_dispatched;  /* siblings suppressed while WAITING or READY */
  uint64_t barrier_in_flight;       /* siblings suppressed while IN-FLIGHT */
  uint64_t queue_dropped;           /* suppressed Grains removed from a Ready Queue */
  uint64_t retried;                 /* Grains moved back to READY at a new generation */
  uint64_t retry_skipped;           /* retry entries naming no in-flight Grain of the Call */
} or_stats;

or_ctx* or_ctx_create(uint32_t n_calls);
void    or_ctx_destroy(or_ctx* ctx);
void    or_ctx_reset(or_ctx* ctx);
void    or_ctx_stats(const or_ctx* ctx, or_stats* out);

/* Expansion (Section 4.2): offsets = exclusive prefix sum of counts, one
 * child per (parent, ordinal) numbered parent-major; empty expansions are
 * terminal at once and listed (ascending) in empty_parents. */
int or_expand(or_ctx* ctx, int32_t parent_xid, const uint32_t* counts, uint64_t n_parents,
              const uint8_t* parent_call, uint64_t* offsets, uint32_t* child_parent,
              uint32_t* child_ordinal, uint64_t child_cap, uint32_t* empty_parents,
              uint64_t* n_children, uint64_t* n_empty, int32_t* xid);

/* Per-Call FIFO Ready Queue with elastic reservation (Section 4.3, Eq. 2).
 * Queued Grains that a GroupFailure suppressed leave the queue at the next
 * reservation without being dispatched (Section 4.4). */
int or_batch_ready(or_ctx* ctx, int32_t xid, uint32_t call, const uint32_t* cand,
                   uint64_t n_cand, uint32_t batch_size, int32_t flush, uint32_t* batched,
                   uint64_t batched_cap, uint64_t* n_batched, uint64_t* n_batches);

/* Parent-bound reservation (Section 4.3): admission as or_batch_ready, then
 * reservations that each take up to B queued siblings of the parent of the
 * queue's first entry (queue order), leaving the other entries in order;
 * repeated while a whole batch of B siblings is at hand (flush: until the
 * queue is empty).  batched gets the batches back to back; batch_off (or
 * NULL) n_batches + 1 boundaries, batch k = batched[batch_off[k] ..
 * batch_off[k+1]).  OR_E_CAPACITY (nothing changes but the queue prelude)
 * when batched_cap or batch_off_cap is too small. */
int or_batch_ready_parent(or_ctx* ctx, int32_t xid, uint32_t call, const uint32_t* cand,
                          uint64_t n_cand, uint32_t batch_size, int32_t flush,
                          uint32_t* batched, uint64_t batched_cap, uint64_t* batch_off,
                          uint64_t batch_off_cap, uint64_t* n_batched, uint64_t* n_batches);

/* Retry of a failed physical attempt (Section 4.4; Eq. 2 IN-FLIGHT -> READY;
 * Section 4.3 recovery queues): each listed Grain of this Call that is
 * IN-FLIGHT (first occurrence in the list) goes back to READY with its
 * generation + 1, and the listed Grains, in list order, form one group in
 * the Call's recovery queue.  The next reservation takes recovery groups,
 * oldest first, before the Ready Queue's entries. */
int or_retry(or_ctx* ctx, int32_t xid, uint32_t call, const uint32_t* children, uint64_t n,
             uint64_t* n_retried);

/* Generation-fenced commit (Section 4.4, Eq. 3) and parent completion
 * (Section 4.2, Reduce); completed parents listed ascending.  An accepted
 * OR_GROUP_FAILURE report seals its Grain Failed and then suppresses every
 * sibling not yet sealed (Section 4.4, Figure 5). */
int or_gather_commit(or_ctx* ctx, int32_t xid, uint64_t n, const uint32_t* child,
                     const uint8_t* state, const uint32_t* len, const uint64_t* off,
                     const uint32_t* gen, uint64_t arena_bytes, uint8_t* code,
                     uint32_t* done_parents, uint64_t done_cap, uint64_t* n_done);

/* Ordered Reduce output (Section 4.2): parents == NULL assembles the parents
 * completed by the latest commit on xid.  With arena and out both NULL only
 * the outcomes and offsets are produced (no bytes copied). */
int or_assemble(or_ctx* ctx, int32_t xid, const uint8_t* arena, uint64_t arena_bytes,
                const uint32_t* parents, uint64_t n_parents, uint8_t* status,
                uint64_t* out_off, uint32_t* out_len, uint8_t* out, uint64_t out_cap,
                uint64_t* out_cursor, uint64_t* out_bytes, uint64_t* n_assembled);

/* List-structured Reduce output (Section 4.2: present values in ordinal
 * order; Table 3's F.reduce gathers a list).  Same as or_assemble, plus for
 * every listed parent that is assembled Present the entries of its members
 * in ordinal order: elem_base[i] .. elem_base[i+1] (elem_base has n+1
 * entries); for each entry its outcome (PRESENT or DROPPED), the output
 * offset of its bytes and their length (0 if Dropped).  Suppressed and
 * incomplete parents have no entries.  elem_cap bounds the entries. */
int or_assemble_list(or_ctx* ctx, int32_t xid, const uint8_t* arena, uint64_t arena_bytes,
                     const uint32_t* parents, uint64_t n_parents, uint8_t* status,
                     uint64_t* out_off, uint32_t* out_len, uint8_t* out, uint64_t out_cap,
                     uint64_t* out_cursor, uint64_t* out_bytes, uint64_t* n_assembled,
                     uint64_t* elem_base, uint8_t* elem_state, uint64_t* elem_off,
                     uint32_t* elem_len, uint64_t elem_cap, uint64_t* n_elems);

/* Bytes and list entries an assembly of `parents` (NULL: the latest commit's
 * completed parents) would produce; changes nothing (no counters). */
int or_assemble_size(or_ctx* ctx, int32_t xid, const uint32_t* parents, uint64_t n_parents,
                     uint64_t* bytes, uint64_t* elems);

/* F.filter (Table 3; Section 4.2's propagation rule) applied to a batch of
 * reports: a Present report whose mask is 0 becomes Dropped; every other
 * report keeps its state (a failed or suppressed input stays so). */
void or_filter_reports(uint8_t* state, const uint8_t* keep, uint64_t n);

#ifdef __cplusplus
}
#endif
#endif
