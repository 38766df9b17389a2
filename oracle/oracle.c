/*
 * oracle.c — plain, single-threaded CPU implementation of RayOrch's lineage
 * expand / FIFO batch / gather-commit / assemble semantics
 * (arXiv 2609.18703, Section 4).
 *
 * TEST INFRASTRUCTURE ONLY: used by the tests, the smoke check and the
 * benchmark's CPU-baseline leg.  It is deliberately naive — one loop per
 * definition, in the order the paper states it, no blocking or fusion — so
 * that it can be read against the paper.  It shares nothing with the GPU
 * library.
 *
 * Where the paper leaves a detail open the reading used is the one listed in
 * the design notes (child numbering parent-major, completed parents reported
 * in ascending id, reports of one commit applied in array order, etc.).
 */
#include "oracle.h"

#include <stdlib.h>
#include <string.h>

#define OR_MAX_EXP 64

typedef struct {
  int32_t parent_xid;
  uint64_t P, N;
  uint64_t* offsets;        /* P+1: exclusive prefix sum of counts */
  uint32_t* child_parent;   /* N: immediate parent of each child */
  uint8_t* child_call;      /* N: the Call whose Grain the child is */
  uint8_t* phase;           /* N: Eq. (2) phase of the child's Grain */
  uint32_t* gen;            /* N: attempt generation of the Grain */
  uint8_t* st;              /* N: published outcome (Eq. 1) */
  uint32_t* len;            /* N: payload length of a Present value */
  uint64_t* off;            /* N: arena offset of a Present value */
  uint8_t* by_barrier;      /* N: sealed by a sibling's GroupFailure */
  uint64_t* terminal;       /* P: members whose outcome has been published */
  uint8_t* bad;             /* P: a member is Failed or Suppressed */
  uint8_t* barrier;         /* P: a GroupFailure suppressed the parent's open members */
  uint32_t** q;             /* per Call: FIFO Ready Queue storage (N slots) */
  uint64_t* qhead;
  uint64_t* qtail;
  uint32_t** rq;            /* per Call: recovery queue (retried Grains, N slots) */
  uint64_t* rlen;
  uint32_t* last_done;      /* parents completed by the latest commit */
  uint64_t n_last_done;
} or_exp;

struct or_ctx {
  uint32_t n_calls;
  int32_t n_exp;
  or_exp* exp[OR_MAX_EXP];
  or_stats stats;
};

static void exp_free(or_exp* x) {
  if (!x) return;
  free(x->offsets); free(x->child_parent); free(x->child_call); free(x->phase);
  free(x->gen); free(x->st); free(x->len); free(x->off); free(x->terminal); free(x->bad);
  free(x->by_barrier); free(x->barrier); free(x->last_done);
  free(x);
}

or_ctx* or_ctx_create(uint32_t n_calls) {
  if (n_calls == 0 || n_calls > 256) return NULL;
  or_ctx* ctx = (or_ctx*)calloc(1, sizeof(or_ctx));
  if (!ctx) return NULL;
  ctx->n_calls = n_calls;
  return ctx;
}

void or_ctx_reset(or_ctx* ctx) {
  if (!ctx) return;
  for (int32_t i = 0; i < ctx->n_exp; ++i) {
    or_exp* x = ctx->exp[i];
    if (x && x->q) {
      for (uint32_t c = 0; c < ctx->n_calls; ++c) free(x->q[c]);
      free(x->q); free(x->qhead); free(x->qtail);
    }
    if (x && x->rq) {
      for (uint32_t c = 0; c < ctx->n_calls; ++c) free(x->rq[c]);
      free(x->rq); free(x->rlen);
    }
    exp_free(x);
    ctx->exp[i] = NULL;
  }
  ctx->n_exp = 0;
}

void or_ctx_destroy(or_ctx* ctx) {
  if (!ctx) return;
  or_ctx_reset(ctx);
  free(ctx);
}

void or_ctx_stats(const or_ctx* ctx, or_stats* out) {
  if (ctx && out) *out = ctx->stats;
}

static or_exp* get_exp(or_ctx* ctx, int32_t xid) {
  if (!ctx || xid < 0 || xid >= ctx->n_exp) return NULL;
  return ctx->exp[xid];
}

static uint64_t member_count(const or_exp* x, uint64_t p) {
  return x->offsets[p + 1] - x->offsets[p];
}

/* ------------------------------------------------------------------------ */
/* Expansion (Section 4.2; Table 2 for the child key): every parent gets its
 * own ordered list of children, each child keyed by (parent, ordinal) with
 * ordinals 0..m-1.  A parent whose list is empty is already resolved
 * (Eq. 1 lists the empty list as a terminal Expansion fact).               */
int or_expand(or_ctx* ctx, int32_t parent_xid, const uint32_t* counts, uint64_t n_parents,
              const uint8_t* parent_call, uint64_t* offsets, uint32_t* child_parent,
              uint32_t* child_ordinal, uint64_t child_cap, uint32_t* empty_parents,
              uint64_t* n_children, uint64_t* n_empty, int32_t* xid) {
  if (!ctx || !xid || !n_children || (n_parents && !counts) || !offsets) return OR_E_INVAL;
  if (ctx->n_exp >= OR_MAX_EXP) return OR_E_INVAL;
  if (n_parents >= ((uint64_t)1 << 32)) return OR_E_OVERFLOW;
  if (parent_xid >= 0) {
    or_exp* px = get_exp(ctx, parent_xid);
    if (!px || px->N != n_parents) return OR_E_INVAL;
  } else if (parent_xid != -1) {
    return OR_E_INVAL;
  }
  if (parent_call) {
    for (uint64_t p = 0; p < n_parents; ++p)
      if (parent_call[p] >= ctx->n_calls) return OR_E_INVAL;
  }

  /* offsets[p] = sum of counts[q] for q < p */
  offsets[0] = 0;
  for (uint64_t p = 0; p < n_parents; ++p) offsets[p + 1] = offsets[p] + counts[p];
  uint64_t N = offsets[n_parents];
  *n_children = N;
  uint64_t ne = 0;
  for (uint64_t p = 0; p < n_parents; ++p) ne += (counts[p] == 0);
  if (n_empty) *n_empty = ne;
  if (N >= ((uint64_t)1 << 32)) return OR_E_OVERFLOW;
  if (N > child_cap) return OR_E_CAPACITY;
  if (N && (!child_parent || !child_ordinal)) return OR_E_INVAL;

  or_exp* x = (or_exp*)calloc(1, sizeof(or_exp));
  if (!x) return OR_E_OOM;
  x->parent_xid = parent_xid;
  x->P = n_parents;
  x->N = N;
  x->offsets = (uint64_t*)malloc((n_parents + 1) * sizeof(uint64_t));
  x->child_parent = (uint32_t*)malloc((N ? N : 1) * sizeof(uint32_t));
  x->child_call = (uint8_t*)malloc(N ? N : 1);
  x->phase = (uint8_t*)malloc(N ? N : 1);
  x->gen = (uint32_t*)malloc((N ? N : 1) * sizeof(uint32_t));
  x->st = (uint8_t*)malloc(N ? N : 1);
  x->len = (uint32_t*)malloc((N ? N : 1) * sizeof(uint32_t));
  x->off = (uint64_t*)malloc((N ? N : 1) * sizeof(uint64_t));
  x->terminal = (uint64_t*)calloc(n_parents ? n_parents : 1, sizeof(uint64_t));
  x->bad = (uint8_t*)calloc(n_parents ? n_parents : 1, 1);
  x->barrier = (uint8_t*)calloc(n_parents ? n_parents : 1, 1);
  x->by_barrier = (uint8_t*)calloc(N ? N : 1, 1);
  x->last_done = (uint32_t*)malloc((n_parents ? n_parents : 1) * sizeof(uint32_t));
  x->q = (uint32_t**)calloc(ctx->n_calls, sizeof(uint32_t*));
  x->qhead = (uint64_t*)calloc(ctx->n_calls, sizeof(uint64_t));
  x->qtail = (uint64_t*)calloc(ctx->n_calls, sizeof(uint64_t));
  x->rq = (uint32_t**)calloc(ctx->n_calls, sizeof(uint32_t*));
  x->rlen = (uint64_t*)calloc(ctx->n_calls, sizeof(uint64_t));
  if (!x->offsets || !x->child_parent || !x->child_call || !x->phase || !x->gen || !x->st ||
      !x->len || !x->off || !x->terminal || !x->bad || !x->barrier || !x->by_barrier ||
      !x->last_done || !x->q || !x->qhead || !x->qtail || !x->rq || !x->rlen) {
    free(x->q); free(x->qhead); free(x->qtail); free(x->rq); free(x->rlen);
    exp_free(x);
    return OR_E_OOM;
  }
  memcpy(x->offsets, offsets, (n_parents + 1) * sizeof(uint64_t));

  /* child c = (parent p, ordinal j), numbered parent-major */
  uint64_t c = 0;
  for (uint64_t p = 0; p < n_parents; ++p) {
    for (uint32_t j = 0; j < counts[p]; ++j) {
      child_parent[c] = (uint32_t)p;
      child_ordinal[c] = j;
      x->child_parent[c] = (uint32_t)p;
      x->child_call[c] = parent_call ? parent_call[p] : 0;
      x->phase[c] = OR_WAITING;
      x->gen[c] = 0;
      x->st[c] = OR_PENDING;
      x->len[c] = 0;
      x->off[c] = 0;
      ++c;
    }
  }

  /* empty Expansions are terminal immediately (listed ascending) */
  uint64_t k = 0;
  for (uint64_t p = 0; p < n_parents; ++p)
    if (counts[p] == 0) {
      if (empty_parents) empty_parents[k] = (uint32_t)p;
      ++k;
    }

  ctx->exp[ctx->n_exp] = x;
  *xid = ctx->n_exp;
  ctx->n_exp++;
  return OR_OK;
}

/* ------------------------------------------------------------------------ */
/* Per-Call FIFO Ready Queue (Section 4.3, Eq. 2).  Candidates are admitted
 * in the order given, WAITING -> READY, if they belong to this Call.  What
 * precedes a reservation of either policy: recovery groups move ahead of the
 * queue's entries, queued Grains sealed since (GroupFailure) leave, and the
 * candidates are admitted behind the tail.  *old_tail gets the tail before
 * admission (to undo it), *bad_cand the candidates naming no child.        */
static int ready_admit(or_ctx* ctx, or_exp* x, uint32_t call, const uint32_t* cand,
                       uint64_t n_cand, uint64_t* old_tail, uint64_t* bad_cand) {
  if (!cand) n_cand = x->N;
  if (!x->q[call]) {
    x->q[call] = (uint32_t*)malloc((x->N ? x->N : 1) * sizeof(uint32_t));
    if (!x->q[call]) return OR_E_OOM;
  }
  uint32_t* q = x->q[call];

  /* recovery groups go first: they are placed ahead of the queue's entries
     (the slots before the head are free: every retried Grain was taken out
     of this queue once) */
  if (x->rlen[call]) {
    uint64_t nr = x->rlen[call];
    if (nr > x->qhead[call]) return OR_E_STATE;   /* cannot happen: see above */
    x->qhead[call] -= nr;
    memcpy(q + x->qhead[call], x->rq[call], nr * sizeof(uint32_t));
    x->rlen[call] = 0;
  }

  /* queued Grains a GroupFailure sealed leave the queue undispatched */
  uint64_t kept = x->qhead[call];
  for (uint64_t t = x->qhead[call]; t < x->qtail[call]; ++t) {
    if (x->phase[q[t]] == OR_READY)
      q[kept++] = q[t];
    else
      ctx->stats.queue_dropped++;
  }
  x->qtail[call] = kept;
  *old_tail = x->qtail[call];

  /* admission: candidates in order; only WAITING Grains of this Call enter */
  uint64_t bad = 0;
  for (uint64_t i = 0; i < n_cand; ++i) {
    uint64_t c = cand ? cand[i] : i;
    if (c >= x->N) { ++bad; continue; }
    if (x->phase[c] != OR_WAITING) continue;
    if (x->child_call[c] != call) continue;
    x->phase[c] = OR_READY;
    q[x->qtail[call]++] = (uint32_t)c;
  }
  *bad_cand = bad;
  return OR_OK;
}

/* Undo an admission (a reservation that did not fit): the call can be
 * repeated with more room. */
static void ready_unadmit(or_exp* x, uint32_t call, uint64_t old_tail) {
  uint32_t* q = x->q[call];
  for (uint64_t t = old_tail; t < x->qtail[call]; ++t) x->phase[q[t]] = OR_WAITING;
  x->qtail[call] = old_tail;
}

/* Elastic reservation takes up to B queued Grains at a time from the front,
 * whatever their parents, READY -> IN-FLIGHT.  Only whole batches are taken,
 * except on flush, which also takes the last partial batch.                */
int or_batch_ready(or_ctx* ctx, int32_t xid, uint32_t call, const uint32_t* cand,
                   uint64_t n_cand, uint32_t batch_size, int32_t flush, uint32_t* batched,
                   uint64_t batched_cap, uint64_t* n_batched, uint64_t* n_batches) {
  or_exp* x = get_exp(ctx, xid);
  if (!x || call >= ctx->n_calls || batch_size == 0) return OR_E_INVAL;
  uint64_t old_tail, bad_cand;
  int rc = ready_admit(ctx, x, call, cand, n_cand, &old_tail, &bad_cand);
  if (rc != OR_OK) return rc;
  uint32_t* q = x->q[call];

  /* reservation: whole batches of B from the head (all on flush) */
  uint64_t queued = x->qtail[call] - x->qhead[call];
  uint64_t take = flush ? queued : (queued / batch_size) * batch_size;
  if (n_batched) *n_batched = take;
  if (take > batched_cap || (take && !batched)) {
    ready_unadmit(x, call, old_tail);
    return take > batched_cap ? OR_E_CAPACITY : OR_E_INVAL;
  }
  for (uint64_t i = 0; i < take; ++i) {
    uint32_t c = q[x->qhead[call] + i];
    batched[i] = c;
    x->phase[c] = OR_IN_FLIGHT;
  }
  x->qhead[call] += take;
  if (n_batches) *n_batches = (take + batch_size - 1) / batch_size;
  ctx->stats.ready_bad_candidates += bad_cand;
  return OR_OK;
}

/* Parent-bound reservation (Section 4.3): one reservation takes up to B
 * queued siblings of the parent of the queue's first entry, in queue order;
 * every entry it leaves keeps its place relative to the others.
 * Reservations repeat while they can be made.  Without flush a reservation
 * that would hold fewer than B siblings is not made, and the queue waits
 * for more of that parent's siblings (as elastic reservation waits for a
 * whole batch); with flush reservations repeat until the queue is empty.
 * Kept as the steps read: the queue is a doubly linked list in queue order
 * and each parent's queued entries a singly linked list in queue order.   */
int or_batch_ready_parent(or_ctx* ctx, int32_t xid, uint32_t call, const uint32_t* cand,
                          uint64_t n_cand, uint32_t batch_size, int32_t flush,
                          uint32_t* batched, uint64_t batched_cap, uint64_t* batch_off,
                          uint64_t batch_off_cap, uint64_t* n_batched, uint64_t* n_batches) {
  or_exp* x = get_exp(ctx, xid);
  if (!x || call >= ctx->n_calls || batch_size == 0) return OR_E_INVAL;
  uint64_t old_tail, bad_cand;
  int rc = ready_admit(ctx, x, call, cand, n_cand, &old_tail, &bad_cand);
  if (rc != OR_OK) return rc;
  uint32_t* q = x->q[call];
  const uint64_t h = x->qhead[call], n = x->qtail[call] - h;

  int64_t* prev = (int64_t*)malloc((n ? n : 1) * sizeof(int64_t));
  int64_t* next = (int64_t*)malloc((n ? n : 1) * sizeof(int64_t));
  int64_t* sib = (int64_t*)malloc((n ? n : 1) * sizeof(int64_t));
  int64_t* first = (int64_t*)malloc((x->P ? x->P : 1) * sizeof(int64_t));
  int64_t* last = (int64_t*)malloc((x->P ? x->P : 1) * sizeof(int64_t));
  uint32_t* out = (uint32_t*)malloc((n ? n : 1) * sizeof(uint32_t));
  uint64_t* bo = (uint64_t*)malloc((n + 1) * sizeof(uint64_t));
  const uint64_t pick_cap = batch_size < n ? batch_size : n;   /* a batch never exceeds the queue */
  int64_t* pick = (int64_t*)malloc((pick_cap ? pick_cap : 1) * sizeof(int64_t));
  if (!prev || !next || !sib || !first || !last || !out || !bo || !pick) {
    free(prev); free(next); free(sib); free(first); free(last); free(out); free(bo); free(pick);
    ready_unadmit(x, call, old_tail);
    return OR_E_OOM;
  }
  for (uint64_t p = 0; p < x->P; ++p) first[p] = last[p] = -1;
  for (uint64_t i = 0; i < n; ++i) {
    prev[i] = (int64_t)i - 1;
    next[i] = i + 1 < n ? (int64_t)i + 1 : -1;
    sib[i] = -1;
    uint32_t p = x->child_parent[q[h + i]];
    if (first[p] < 0) first[p] = (int64_t)i; else sib[last[p]] = (int64_t)i;
    last[p] = (int64_t)i;
  }
  int64_t front = n ? 0 : -1;
  uint64_t take = 0, nb = 0;
  while (front >= 0) {
    /* the first ready parent: the parent of the queue's first entry */
    uint32_t p = x->child_parent[q[h + front]];
    uint64_t k = 0;
    int64_t e = first[p];
    while (e >= 0 && k < batch_size) { pick[k++] = e; e = sib[e]; }
    if (k < batch_size && !flush) break;   /* short of B: wait for more siblings */
    bo[nb++] = take;
    for (uint64_t j = 0; j < k; ++j) {
      int64_t t = pick[j];
      out[take++] = q[h + t];
      if (prev[t] >= 0) next[prev[t]] = next[t]; else front = next[t];
      if (next[t] >= 0) prev[next[t]] = prev[t];
    }
    first[p] = e;
  }
  bo[nb] = take;

  if (n_batched) *n_batched = take;
  if (n_batches) *n_batches = nb;
  int bad = take > batched_cap ? OR_E_CAPACITY
          : (batch_off && nb + 1 > batch_off_cap) ? OR_E_CAPACITY
          : (take && !batched) ? OR_E_INVAL : OR_OK;
  if (bad != OR_OK) {
    ready_unadmit(x, call, old_tail);
  } else {
    for (uint64_t i = 0; i < take; ++i) {
      batched[i] = out[i];
      x->phase[out[i]] = OR_IN_FLIGHT;
    }
    if (batch_off) memcpy(batch_off, bo, (nb + 1) * sizeof(uint64_t));
    /* the entries left, in queue order, behind the new head */
    uint64_t r = 0;
    for (int64_t t = front; t >= 0; t = next[t]) out[r++] = q[h + t];
    memcpy(q + h + take, out, r * sizeof(uint32_t));
    x->qhead[call] = h + take;
    ctx->stats.ready_bad_candidates += bad_cand;
  }
  free(prev); free(next); free(sib); free(first); free(last); free(out); free(bo); free(pick);
  return bad;
}

/* ------------------------------------------------------------------------ */
/* Retry (Section 4.4; Eq. 2's IN-FLIGHT -> READY edge).  A physical attempt
 * failed: its Grains keep their identity, return to READY with the next
 * generation (so reports of the failed attempt are stale), and re-enter as
 * one group of the Call's recovery queue, ahead of normal entries
 * (Section 4.3).                                                           */
int or_retry(or_ctx* ctx, int32_t xid, uint32_t call, const uint32_t* children, uint64_t n,
             uint64_t* n_retried) {
  or_exp* x = get_exp(ctx, xid);
  if (!x || call >= ctx->n_calls || (n && !children)) return OR_E_INVAL;
  if (!x->rq[call]) {
    x->rq[call] = (uint32_t*)malloc((x->N ? x->N : 1) * sizeof(uint32_t));
    if (!x->rq[call]) return OR_E_OOM;
  }
  uint64_t k = 0;
  for (uint64_t i = 0; i < n; ++i) {
    uint64_t c = children[i];
    if (c >= x->N || x->phase[c] != OR_IN_FLIGHT || x->child_call[c] != call) {
      ctx->stats.retry_skipped++;
      continue;
    }
    x->phase[c] = OR_READY;
    x->gen[c] += 1;
    x->rq[call][x->rlen[call]++] = (uint32_t)c;
    ++k;
  }
  ctx->stats.retried += k;
  if (n_retried) *n_retried = k;
  return OR_OK;
}

static int cmp_u32(const void* a, const void* b) {
  uint32_t x = *(const uint32_t*)a, y = *(const uint32_t*)b;
  return (x > y) - (x < y);
}

/* ------------------------------------------------------------------------ */
/* Commit (Section 4.4, Eq. 3).  The fence admits a report when the child's
 * Grain is IN-FLIGHT and the report carries the Grain's current generation;
 * an admitted report moves the Grain to SEALED and records its outcome
 * (Eq. 1), after which nothing can change it.  A parent is complete once all
 * of its children have a recorded outcome (Section 4.2, Reduce).  Reports
 * are applied one after another in array order.  A GroupFailure report
 * (Section 4.4, Figure 5) fails its own Grain and then suppresses the
 * parent's other open Grains: queued ones will never be dispatched, and the
 * later reports of in-flight ones are rejected.                            */
int or_gather_commit(or_ctx* ctx, int32_t xid, uint64_t n, const uint32_t* child,
                     const uint8_t* state, const uint32_t* len, const uint64_t* off,
                     const uint32_t* gen, uint64_t arena_bytes, uint8_t* code,
                     uint32_t* done_parents, uint64_t done_cap, uint64_t* n_done) {
  or_exp* x = get_exp(ctx, xid);
  if (!x || (n && (!child || !state || !len || !off))) return OR_E_INVAL;
  uint64_t need = n < x->P ? n : x->P;
  if (done_parents && done_cap < need) return OR_E_INVAL;

  uint64_t k = 0;
  for (uint64_t r = 0; r < n; ++r) {
    uint64_t c = child[r];
    uint8_t s = state[r];
    uint32_t g = gen ? gen[r] : 0;
    uint8_t v;
    int valid_state = (s == OR_PRESENT || s == OR_DROPPED || s == OR_FAILED ||
                       s == OR_SUPPRESSED || s == OR_GROUP_FAILURE);
    int in_bounds = (s != OR_PRESENT) || (off[r] <= arena_bytes && len[r] <= arena_bytes - off[r]);
    if (c >= x->N || !valid_state || !in_bounds) {
      v = OR_REJ_INVALID;
    } else if (x->phase[c] == OR_WAITING || x->phase[c] == OR_READY) {
      v = OR_REJ_NOT_INFLIGHT;
    } else if (g != x->gen[c]) {
      v = OR_REJ_STALE_GEN;
    } else if (x->phase[c] == OR_SEALED) {
      v = x->by_barrier[c] ? OR_REJ_BARRIER : OR_REJ_DUPLICATE;
    } else {
      v = OR_ACCEPT;
      x->phase[c] = OR_SEALED;
      x->st[c] = (s == OR_GROUP_FAILURE) ? OR_FAILED : s;   /* the reporting Grain failed */
      x->len[c] = (s == OR_PRESENT) ? len[r] : 0;
      x->off[c] = (s == OR_PRESENT) ? off[r] : 0;
      uint32_t p = x->child_parent[c];
      x->terminal[p] += 1;
      if (s == OR_FAILED || s == OR_SUPPRESSED || s == OR_GROUP_FAILURE) x->bad[p] = 1;
      if (x->terminal[p] == member_count(x, p)) x->last_done[k++] = p;
      if (s == OR_GROUP_FAILURE && !x->barrier[p]) {
        /* the barrier for (Call, parent): every sibling not yet sealed is
           suppressed now, queued or in flight; sealed ones keep their facts */
        x->barrier[p] = 1;
        uint64_t sealed_now = 0;
        for (uint64_t d = x->offsets[p]; d < x->offsets[p + 1]; ++d) {
          if (x->phase[d] == OR_SEALED) continue;
          if (x->phase[d] == OR_IN_FLIGHT)
            ctx->stats.barrier_in_flight++;
          else
            ctx->stats.barrier_not_dispatched++;
          x->phase[d] = OR_SEALED;
          x->st[d] = OR_SUPPRESSED;
          x->len[d] = 0;
          x->off[d] = 0;
          x->by_barrier[d] = 1;
          x->terminal[p] += 1;
          ++sealed_now;
        }
        if (sealed_now && x->terminal[p] == member_count(x, p)) x->last_done[k++] = p;
      }
    }
    if (code) code[r] = v;
    switch (v) {
      case OR_ACCEPT: ctx->stats.accepted++; break;
      case OR_REJ_INVALID: ctx->stats.rej_invalid++; break;
      case OR_REJ_NOT_INFLIGHT: ctx->stats.rej_not_inflight++; break;
      case OR_REJ_STALE_GEN: ctx->stats.rej_stale_gen++; break;
      case OR_REJ_BARRIER: ctx->stats.rej_barrier++; break;
      default: ctx->stats.rej_duplicate++; break;
    }
  }
  qsort(x->last_done, k, sizeof(uint32_t), cmp_u32);
  x->n_last_done = k;
  if (done_parents) memcpy(done_parents, x->last_done, k * sizeof(uint32_t));
  if (n_done) *n_done = k;
  return OR_OK;
}

/* ------------------------------------------------------------------------ */
/* Reduce output (Section 4.2).  If any child of a completed parent Failed or
 * was Suppressed, the parent is Suppressed and contributes no bytes.
 * Otherwise the parent is Present and its value is the concatenation, by
 * ordinal, of its Present children's payloads; Dropped children add nothing,
 * so a parent whose children were all Dropped is Present with 0 bytes.
 * Parents are written back to back from the cursor (or 0) in list order.   */
int or_assemble(or_ctx* ctx, int32_t xid, const uint8_t* arena, uint64_t arena_bytes,
                const uint32_t* parents, uint64_t n_parents, uint8_t* status,
                uint64_t* out_off, uint32_t* out_len, uint8_t* out, uint64_t out_cap,
                uint64_t* out_cursor, uint64_t* out_bytes, uint64_t* n_assembled) {
  or_exp* x = get_exp(ctx, xid);
  if (!x || !status || !out_off) return OR_E_INVAL;
  const uint32_t* list = parents ? parents : x->last_done;
  uint64_t n = parents ? n_parents : x->n_last_done;
  if (n_assembled) *n_assembled = n;
  if (!parents && n > n_parents) return OR_E_CAPACITY;
  uint64_t base = out_cursor ? *out_cursor : 0;

  /* sizes first, so that nothing is written when the output cannot hold it */
  uint64_t total = 0;
  int len_overflow = 0;
  for (uint64_t i = 0; i < n; ++i) {
    uint64_t p = list[i];
    if (p >= x->P || x->terminal[p] != member_count(x, p) || x->bad[p]) continue;
    uint64_t bytes = 0;
    for (uint64_t c = x->offsets[p]; c < x->offsets[p + 1]; ++c)
      if (x->st[c] == OR_PRESENT) bytes += x->len[c];
    if (bytes > 0xFFFFFFFFull) len_overflow = 1;
    total += bytes;
  }
  if (out_bytes) *out_bytes = total;
  if (base + total > out_cap) return OR_E_CAPACITY;
  if (out_len && len_overflow) return OR_E_OVERFLOW;
  /* arena and out both NULL: outcomes and offsets only, no bytes copied */
  const int sizes_only = !out && !arena;
  if (total && !sizes_only && (!out || !arena)) return OR_E_INVAL;

  uint64_t pos = base;
  for (uint64_t i = 0; i < n; ++i) {
    uint64_t p = list[i];
    uint64_t start = pos;
    if (p >= x->P || x->terminal[p] != member_count(x, p)) {
      status[i] = OR_PENDING;
      ctx->stats.assemble_incomplete++;
    } else if (x->bad[p]) {
      status[i] = OR_SUPPRESSED;
    } else {
      status[i] = OR_PRESENT;
      for (uint64_t c = x->offsets[p]; c < x->offsets[p + 1]; ++c) {
        if (x->st[c] != OR_PRESENT) continue;   /* Dropped members are excluded */
        if (!sizes_only) memcpy(out + pos, arena + x->off[c], x->len[c]);
        pos += x->len[c];
      }
    }
    out_off[i] = start;
    if (out_len) out_len[i] = (uint32_t)(pos - start);
  }
  out_off[n] = pos;
  if (out_cursor) *out_cursor = pos;
  (void)arena_bytes;
  return OR_OK;
}

/* ------------------------------------------------------------------------ */
/* List-structured Reduce output (Section 4.2): the parent's value is the
 * list of its present members' values in ordinal order; the entries below
 * let a reader split the concatenated bytes back into that list.  Dropped
 * members are listed with their outcome and no bytes.                      */
int or_assemble_list(or_ctx* ctx, int32_t xid, const uint8_t* arena, uint64_t arena_bytes,
                     const uint32_t* parents, uint64_t n_parents, uint8_t* status,
                     uint64_t* out_off, uint32_t* out_len, uint8_t* out, uint64_t out_cap,
                     uint64_t* out_cursor, uint64_t* out_bytes, uint64_t* n_assembled,
                     uint64_t* elem_base, uint8_t* elem_state, uint64_t* elem_off,
                     uint32_t* elem_len, uint64_t elem_cap, uint64_t* n_elems) {
  or_exp* x = get_exp(ctx, xid);
  if (!x || !elem_base) return OR_E_INVAL;
  const uint32_t* list = parents ? parents : x->last_done;
  uint64_t n = parents ? n_parents : x->n_last_done;
  uint64_t base = out_cursor ? *out_cursor : 0;
  /* entries first: the members of every listed parent that is complete and
     not suppressed */
  uint64_t ne = 0;
  for (uint64_t i = 0; i < n; ++i) {
    uint64_t p = list[i];
    if (p >= x->P || x->terminal[p] != member_count(x, p) || x->bad[p]) continue;
    ne += member_count(x, p);
  }
  if (n_elems) *n_elems = ne;
  if (ne > elem_cap) return OR_E_CAPACITY;
  if (ne && (!elem_state || !elem_off || !elem_len)) return OR_E_INVAL;
  int st = or_assemble(ctx, xid, arena, arena_bytes, parents, n_parents, status, out_off, out_len,
                       out, out_cap, out_cursor, out_bytes, n_assembled);
  if (st != OR_OK) return st;
  uint64_t e = 0, pos = base;
  for (uint64_t i = 0; i < n; ++i) {
    uint64_t p = list[i];
    elem_base[i] = e;
    if (p >= x->P || x->terminal[p] != member_count(x, p) || x->bad[p]) continue;
    for (uint64_t c = x->offsets[p]; c < x->offsets[p + 1]; ++c) {
      elem_state[e] = x->st[c];
      elem_off[e] = pos;
      elem_len[e] = (x->st[c] == OR_PRESENT) ? x->len[c] : 0;
      pos += elem_len[e];
      ++e;
    }
  }
  elem_base[n] = e;
  return OR_OK;
}

/* F.filter (Table 3): pass on true, drop on false; inputs that failed or
 * were suppressed keep their state (Section 4.2's propagation precedence). */
void or_filter_reports(uint8_t* state, const uint8_t* keep, uint64_t n) {
  for (uint64_t r = 0; r < n; ++r)
    if (state[r] == OR_PRESENT && !keep[r]) state[r] = OR_DROPPED;
}

int or_assemble_size(or_ctx* ctx, int32_t xid, const uint32_t* parents, uint64_t n_parents,
                     uint64_t* bytes, uint64_t* elems) {
  or_exp* x = get_exp(ctx, xid);
  if (!x) return OR_E_INVAL;
  const uint32_t* list = parents ? parents : x->last_done;
  uint64_t n = parents ? n_parents : x->n_last_done;
  uint64_t b = 0, e = 0;
  for (uint64_t i = 0; i < n; ++i) {
    uint64_t p = list[i];
    if (p >= x->P || x->terminal[p] != member_count(x, p) || x->bad[p]) continue;
    e += member_count(x, p);
    for (uint64_t c = x->offsets[p]; c < x->offsets[p + 1]; ++c)
      if (x->st[c] == OR_PRESENT) b += x->len[c];
  }
  if (bytes) *bytes = b;
  if (elems) *elems = e;
  return OR_OK;
}
