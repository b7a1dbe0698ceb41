"""The oracle's pins must catch plausible mistakes.

Each case plants one mistake in a temporary copy of ``oracle/oracle.c`` (a
dropped term, a wrong comparison, sign or bound, a lost reset), builds it on
the CPU, routes the oracle wrappers to it and runs a battery of pins drawn from
the other oracle tests.  At least one pin must fail for every planted mistake.
The committed oracle is never modified.
"""
import os
import subprocess

import numpy as np
import pytest

import oracle
import test_oracle_calibration as K
import test_oracle_fragility as F
import test_oracle_rq as R
import test_oracle_search as S
import test_oracle_stopping as T

SRC = os.path.join(os.path.dirname(oracle.__file__), "oracle.c")

MUTATIONS = [
    ("tau test strict", "ix->d);\n        if (s >= tau) {", "ix->d);\n        if (s > tau) {"),
    ("hit does not reset the run", "if (f(ctx, searched))\n            stale = 0;",
     "if (f(ctx, searched))\n            stale = stale;"),
    ("id tie-break reversed", "(sa == sb && ia < ib)", "(sa == sb && ia > ib)"),
    ("stop line one short", "int64_t reach = (int64_t)j + W;", "int64_t reach = (int64_t)j + W - 1;"),
    ("first coordinate dropped", "for (int t = 0; t < d; ++t)\n        acc += (double)a[t]",
     "for (int t = 1; t < d; ++t)\n        acc += (double)a[t]"),
    ("centroid order reversed", "if (x->score > y->score) return -1;",
     "if (x->score > y->score) return 1;"),
    ("self not excluded", "if (has_qid && id == qid)\n            continue;\n        double s = sim64",
     "double s = sim64"),
    ("initial stop line 1", "int64_t s = W < nprobe ? W : nprobe;", "int64_t s = 1;"),
    ("merge drops last local entry", "m < (local_n[j] > 0 ? local_n[j] : 0)",
     "m + 1 < (local_n[j] > 0 ? local_n[j] : 0)"),
    ("window off by one", "while (searched < nprobe && stale < W)",
     "while (searched < nprobe && stale <= W)"),
    ("required window one short", "h[1 + longest]++;", "h[longest > 0 ? longest : 1]++;"),
    ("empty run not reset by a hit", "run = local_n[j - 1] > 0 ? 0 : run + 1;",
     "run = local_n[j - 1] > 0 ? run : run + 1;"),
    ("loss target inclusive", "if (loss < eps) {", "if (loss <= eps) {"),
    ("quantized estimate without the centroid term",
     "return qc + (double)ix->factors[row] * (dot - ix->mid * sq);",
     "return (double)ix->factors[row] * (dot - ix->mid * sq);"),
    ("quantized estimate with the code offset added", "(dot - ix->mid * sq)", "(dot + ix->mid * sq)"),
    ("codes from the untransposed rotation", "acc = fma(P[(int64_t)j * d + t], o[j], acc);",
     "acc = fma(P[(int64_t)t * d + j], o[j], acc);"),
    ("code step half as wide", "const double delta = 2.0 * mx / top;",
     "const double delta = mx / top;"),
    ("query rotated by the untransposed matrix", "acc += P[(int64_t)j * d + t] * (double)q[j];",
     "acc += P[(int64_t)t * d + j] * (double)q[j];"),
    # the divergence tagger: which mismatches the parity tests excuse
    ("k-th gap taken one rank early",
     "kth_gap[i] = (t.n > k) ? fin[k - 1].score - fin[k].score : INFINITY;",
     "kth_gap[i] = (t.n > k) ? fin[k > 1 ? k - 2 : 0].score - fin[k - 1].score : INFINITY;"),
    ("centroid gap over nprobe ranks, not nprobe + 1",
     "int64_t top = (int64_t)nprobe + 1 < nlist ? (int64_t)nprobe + 1 : nlist;",
     "int64_t top = (int64_t)nprobe < nlist ? (int64_t)nprobe : nlist;"),
    ("tau gap counts the query's own row",
     "if (qids && ids[row] == qids[i])\n                        continue;\n"
     "                    double s = rq ? rq_estimate",
     "double s = rq ? rq_estimate"),
]


def _pins(tiny, deep):
    """Each pin is a zero-argument callable that raises on failure."""
    return [
        T.test_golden_examples,
        lambda: T.test_exhaustive_patterns(6),
        S.test_tau_boundary_self_and_ties,
        S.test_fig4_walk_end_to_end,
        lambda: S.test_rank_matches_numpy_sort(tiny),
        lambda: S.test_full_probe_equals_bruteforce(deep),
        lambda: S.test_window_at_least_nprobe_is_fixed_probe(tiny, 16),
        lambda: S.test_probes_follow_hit_pattern(deep),
        lambda: K.test_calibration_matches_brute_force_loss(deep, 0.05),
        lambda: K.test_calibration_window_extremes_and_fallbacks(deep),
        K.test_calibration_histogram_of_gapped_hits,
        R.test_grid_aligned_rows_are_estimated_exactly,
        lambda: R.test_estimator_error_shrinks_with_bits_and_is_unbiased(tiny),
        lambda: R.test_quantized_search_approaches_exact(deep),
        lambda: R.test_rows_at_their_centroid_and_bounds(tiny),
        lambda: F.test_hand_built_gaps(F.hand_index()),
        lambda: F.test_upto_below_nprobe_limits_the_rows(F.hand_index()),
        lambda: F.test_fewer_than_k_plus_one_qualifiers_give_infinity(F.hand_index()),
        F.test_exact_ties_give_zero_gaps,
        lambda: F.test_nlist_at_most_nprobe_plus_one(F.hand_index()),
        lambda: F.test_tags_equal_numpy_restatement(deep, 3),
    ]


@pytest.mark.parametrize("name,old,new", MUTATIONS, ids=[m[0] for m in MUTATIONS])
def test_planted_mistake_is_caught(tmp_path, tiny, deep, name, old, new):
    src = open(SRC).read()
    assert src.count(old) == 1, f"mutation site for '{name}' not unique"
    mutated = tmp_path / "oracle_mut.c"
    mutated.write_text(src.replace(old, new))
    lib = tmp_path / "liboracle_mut.so"
    subprocess.run(["gcc", "-std=c11", "-O2", "-ffp-contract=off", "-fopenmp", "-fPIC", "-shared",
                    "-o", str(lib),
                    str(mutated), "-lm"], check=True)
    oracle.use_library(str(lib))
    failed = []
    try:
        for pin in _pins(tiny, deep):
            try:
                pin()
            except (AssertionError, ValueError):
                failed.append(pin)
    finally:
        oracle.use_library(None)
    assert failed, f"no pin caught the planted mistake '{name}'"
