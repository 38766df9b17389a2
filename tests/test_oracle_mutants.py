"""The oracle's pins must catch plausible mistakes.  Each case plants one
mistake in a private copy of the oracle's C source (on the CPU), builds it,
and runs the pin suite against it; the suite has to fail."""
import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

MUTANTS = {
    "ordinal_off_by_one": ("child_ordinal[c] = j;", "child_ordinal[c] = j + 1;"),
    "flush_ignored": ("uint64_t take = flush ? queued : (queued / batch_size) * batch_size;",
                      "uint64_t take = (queued / batch_size) * batch_size;"),
    "readmits_queued": ("if (x->phase[c] != OR_WAITING) continue;", ";"),
    "admits_other_calls": ("    if (x->child_call[c] != call) continue;\n", "\n"),
    "fence_ignores_generation": ("} else if (g != x->gen[c]) {", "} else if (0) {"),
    "completion_off_by_one": ("if (x->terminal[p] == member_count(x, p)) x->last_done[k++] = p;",
                              "if (x->terminal[p] + 1 == member_count(x, p)) x->last_done[k++] = p;"),
    "dropped_suppresses": ("if (s == OR_FAILED || s == OR_SUPPRESSED || s == OR_GROUP_FAILURE) x->bad[p] = 1;",
                           "if (s != OR_PRESENT) x->bad[p] = 1;"),
    "source_index_shift": ("memcpy(out + pos, arena + x->off[c], x->len[c]);",
                           "memcpy(out + pos, arena + x->off[c] + 1, x->len[c]);"),
    "done_list_unsorted": ("qsort(x->last_done, k, sizeof(uint32_t), cmp_u32);", "(void)cmp_u32;"),
    "len_off_transposed": ("x->off[c] = (s == OR_PRESENT) ? off[r] : 0;",
                           "x->off[c] = (s == OR_PRESENT) ? len[r] : 0;"),
    "scan_extra_term": ("offsets[p + 1] = offsets[p] + counts[p];",
                        "offsets[p + 1] = offsets[p] + counts[p] + (p == 1);"),
    # GroupFailure containment (Section 4.4)
    "barrier_spares_queued": ("if (x->phase[d] == OR_SEALED) continue;",
                              "if (x->phase[d] != OR_IN_FLIGHT) continue;"),
    "barrier_reseals_committed": ("if (x->phase[d] == OR_SEALED) continue;", "if (d == c) continue;"),
    "queue_keeps_suppressed": ("if (x->phase[q[t]] == OR_READY)", "if (1)"),
    "barrier_verdict_lost": ("v = x->by_barrier[c] ? OR_REJ_BARRIER : OR_REJ_DUPLICATE;",
                             "v = OR_REJ_DUPLICATE;"),
    # retry and recovery queues (Section 4.4, Eq. 2; Section 4.3)
    "retry_keeps_generation": ("    x->gen[c] += 1;\n", "    (void)0;\n"),
    "recovery_never_reinserted": ("  if (x->rlen[call]) {", "  if (0) {"),
    "recovery_behind_queue": ("    memcpy(q + x->qhead[call], x->rq[call], nr * sizeof(uint32_t));",
                              "    for (uint64_t i = 0; i < nr; ++i) q[x->qhead[call] + i] = x->rq[call][nr - 1 - i];"),
    "retry_ignores_call": ("if (c >= x->N || x->phase[c] != OR_IN_FLIGHT || x->child_call[c] != call) {",
                           "if (c >= x->N || x->phase[c] != OR_IN_FLIGHT) {"),
    # list-structured output and F.filter (Section 4.2, Table 3)
    "list_state_lost": ("      elem_state[e] = x->st[c];", "      elem_state[e] = OR_PRESENT;"),
    "list_base_off_by_one": ("  elem_base[n] = e;", "  elem_base[n] = e + 1;"),
    "filter_drops_failed": ("if (state[r] == OR_PRESENT && !keep[r]) state[r] = OR_DROPPED;",
                            "if (!keep[r]) state[r] = OR_DROPPED;"),
    # parent-bound reservation (Section 4.3)
    "pb_takes_short_head": ("if (k < batch_size && !flush) break;", "if (0) break;"),
    "pb_mixes_parents": ("while (e >= 0 && k < batch_size) { pick[k++] = e; e = sib[e]; }",
                         "while (e >= 0 && k < batch_size) { pick[k++] = e; e = next[e]; }"),
    "pb_left_reordered": ("for (int64_t t = front; t >= 0; t = next[t]) out[r++] = q[h + t];",
                          "for (int64_t t = front; t >= 0; t = next[t]) out[r++] = q[h + (t ^ 1) % (int64_t)n];"),
    "pb_batch_off_shift": ("    bo[nb++] = take;\n", "    bo[nb++] = take + (nb > 0);\n"),
    "pb_head_from_tail": ("uint32_t p = x->child_parent[q[h + front]];",
                          "uint32_t p = x->child_parent[q[x->qtail[call] - 1]];"),
    "barrier_completion_missed": ("if (sealed_now && x->terminal[p] == member_count(x, p)) x->last_done[k++] = p;",
                                  "(void)sealed_now;"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_catch_planted_mistake(name, tmp_path):
    before, after = MUTANTS[name]
    src = open(os.path.join(ROOT, "oracle", "oracle.c")).read()
    assert src.count(before) == 1, f"mutation site for {name} not unique"
    (tmp_path / "oracle.c").write_text(src.replace(before, after))
    shutil.copy(os.path.join(ROOT, "oracle", "oracle.h"), tmp_path / "oracle.h")
    so = tmp_path / "libmutant.so"
    subprocess.run(["gcc", "-O1", "-std=c11", "-fPIC", "-shared", "-w", "-o", str(so),
                    str(tmp_path / "oracle.c")], check=True)
    env = dict(os.environ, ORACLE_LIB=str(so))
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                        os.path.join(ROOT, "tests", "test_oracle.py"),
                        os.path.join(ROOT, "tests", "test_oracle_group_failure.py"),
                        os.path.join(ROOT, "tests", "test_oracle_retry.py"),
                        os.path.join(ROOT, "tests", "test_oracle_lists.py"),
                        os.path.join(ROOT, "tests", "test_oracle_parent_bound.py")],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode != 0, f"pins did not catch mutant {name}:\n{r.stdout[-2000:]}"
