"""Comparison rules between the CUDA path and the oracle.

Tolerances (bf16 inputs, fp32 accumulation on the device, float64 oracle):
floating outputs (attention, logit statistics, features, probabilities)
must satisfy |gpu - ref| <= 2e-2 + 1e-2 |ref|; ids, accepted lengths,
emitted tokens and the committed cache bytes must be bit-exact, except for
sequences whose discrete outcome hinges on a near tie: an oracle top-1/top-2
logit margin below 1e-3 on a row that decides the round, or a policy
probability within 1e-3 of the threshold at an evaluated mismatch.  Those
sequences are counted and reported, and excluded from the bit-exact checks.
"""
from __future__ import annotations

import numpy as np

TOL_ABS = 2e-2
TOL_REL = 1e-2
TIE = 1e-3


def assert_close(got, ref, what: str, abs_tol: float = TOL_ABS, rel_tol: float = TOL_REL):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, f"{what}: shape {got.shape} vs {ref.shape}"
    nan_ref = np.isnan(ref)
    assert np.array_equal(np.isnan(got), nan_ref), f"{what}: NaN pattern differs"
    g, r = got[~nan_ref], ref[~nan_ref]
    err = np.abs(g - r)
    bad = err > abs_tol + rel_tol * np.abs(r)
    assert not bad.any(), (f"{what}: {bad.sum()} of {bad.size} outside tolerance, "
                           f"max err {err.max():.3e}")
    return float(err.max()) if err.size else 0.0


def tie_positions(ref_stats, ref_draft, ref_argmax, ref_p, s_ref, s_gpu, lam, margin=None):
    """Near-tie positions of each sequence among those that decide its round:
    rows 0..min(K, max(s_oracle, s_gpu)) whose oracle top-1/top-2 margin is
    below TIE, and evaluated mismatches whose policy probability is within
    TIE of lambda.  ref_stats [B,R,5], ref_draft [B,K], ref_argmax [B,R],
    ref_p [B,K], s_* [B].  ``margin`` [B,R] overrides the top-1/top-2 logit
    gap (for sampled candidates: the gap of the perturbed keys).  Returns an
    int array [B] of counts."""
    B, R = ref_argmax.shape
    K = R - 1
    if margin is None:
        margin = ref_stats[:, :, 0] - ref_stats[:, :, 1]
    counts = np.zeros(B, dtype=np.int64)
    for b in range(B):
        reach = min(K, int(max(s_ref[b], s_gpu[b])))
        counts[b] += int(np.sum(margin[b, : reach + 1] < TIE))
        for i in range(1, reach + 1):
            if i <= K and ref_draft[b, i - 1] != ref_argmax[b, i - 1] and abs(ref_p[b, i - 1] - lam) < TIE:
                counts[b] += 1
    return counts


def tie_affected(ref_stats, ref_draft, ref_argmax, ref_p, s_ref, s_gpu, lam, margin=None):
    """Per-sequence tie flags: a sequence with any near-tie position
    (tie_positions) has its discrete outputs excluded from the bit-exact
    comparison."""
    return tie_positions(ref_stats, ref_draft, ref_argmax, ref_p, s_ref, s_gpu, lam, margin) > 0


# (test, workload, tie-affected sequences, sequences, near-tie positions) of
# every parity test that counts ties; printed at the end of the session and,
# when COSPEC_PARITY_REPORT names a file, written there as JSON.
TIE_REPORT = []


def report_ties(test: str, workload: str, counts) -> None:
    counts = np.asarray(counts)
    TIE_REPORT.append({"test": test, "workload": workload,
                       "tie_affected_sequences": int(np.sum(counts > 0)),
                       "sequences": int(counts.size), "tie_positions": int(np.sum(counts))})
