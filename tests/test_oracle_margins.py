"""Pins of the oracle's decision margins.

The end-to-end parity tests certify a unit when every decision the literal
oracle takes there (Algorithm 2's refinement and Algorithm 1's UpdateCache)
compares two scores whose relative gap |a - b| / max(|a|, |b|) is at least
1e-3: the K/K+1 boundary of the native Top-K (Sec. 2), the ranks of Top_R
including its R/R+1 boundary, the argmin over the residents and the strict
test of each refinement candidate against it (Algorithm 2), and the argmin of
every eviction (Algorithm 1).  Each test below builds one access in which
exactly one of those decisions is close (gap g0) and every other gap is wide,
and checks that the reported margin is g0; a close pair that is no decision
must leave the margin wide.  Leaving any decision out of the margin (or
counting a non-decision) fails one of them.
"""
import numpy as np
import pytest

G0 = 1e-4


def _chain(oracle_lib, N, members=(), aT=None):
    ch = oracle_lib.Chain(N)
    ch.in_cache[list(members)] = 1
    ch.count.value = len(members)
    if aT is not None:
        ch.aT[:] = aT
    return ch


def test_topk_boundary_is_the_margin(oracle_lib):
    # ranks 2 and 3 of p^R (K = 2) differ by G0; cold cache: no eviction decision
    pR = [0.30, 0.20, 0.20 * (1 - G0), 0.05, 0.05, 0.05, 0.05, 0.05]
    ch = _chain(oracle_lib, 8)
    topk, mi, pr, mg = oracle_lib.step(ch, 0, K=2, C=3, R=0, pR=pR, pT=[0.0] * 8)
    assert topk == [0, 1] and mi == 2 and pr == 0
    assert mg == pytest.approx(G0, rel=1e-6)


def test_close_scores_below_the_topk_boundary_do_not_count(oracle_lib):
    # ranks 3 and 4 are close but no decision separates them
    pR = [0.30, 0.20, 0.10, 0.10 * (1 - G0), 0.01, 0.01, 0.01, 0.01]
    ch = _chain(oracle_lib, 8)
    _, _, _, mg = oracle_lib.step(ch, 0, K=2, C=3, R=0, pR=pR, pT=[0.0] * 8)
    assert mg == pytest.approx(0.5)               # |0.2 - 0.1| / 0.2


def test_eviction_argmin_is_the_margin(oracle_lib):
    # full cache {0,1,2}, S = {5}: the victim is 1 (s^T 0.2), 2 is G0 above it
    pR = [0.10, 0.10, 0.10, 0.05, 0.05, 0.50, 0.05, 0.05]
    sT = np.array([0.40, 0.20, 0.20 / (1 - G0), 0.1, 0.1, 0.9, 0.1, 0.1])
    pT = sT - np.array(pR)
    ch = _chain(oracle_lib, 8, (0, 1, 2))
    topk, mi, _, mg = oracle_lib.step(ch, 0, K=1, C=3, R=0, pR=pR, pT=pT)
    assert topk == [5] and mi == 1 and ch.members() == {0, 2, 5}
    assert mg == pytest.approx(G0, rel=1e-6)


def test_eviction_among_wide_scores_is_not_close(oracle_lib):
    # same access with the residents' s^T far apart: only wide gaps remain
    pR = [0.10, 0.10, 0.10, 0.05, 0.05, 0.50, 0.05, 0.05]
    sT = np.array([0.40, 0.20, 0.30, 0.1, 0.1, 0.9, 0.1, 0.1])
    ch = _chain(oracle_lib, 8, (0, 1, 2))
    _, _, _, mg = oracle_lib.step(ch, 0, K=1, C=3, R=0, pR=pR, pT=sT - np.array(pR))
    assert mg == pytest.approx(1 / 3)             # |0.2 - 0.3| / 0.3


def _refine_step(oracle_lib, sST, members, R, C=3):
    """One access at t = 1 whose s^ST is given (a^T = s^ST, p^S = 0) and whose
    access is a wide hit on expert 0 (resident in every case)."""
    N = len(sST)
    ch = _chain(oracle_lib, N, members, aT=sST)
    pR = [0.60] + [0.40 / (N - 1)] * (N - 1)
    out = oracle_lib.step(ch, 1, K=1, C=C, R=R, pR=pR, pT=[0.0] * N, pS_pred=[0.0] * N)
    return ch, out


def test_refinement_rank_boundary_is_the_margin(oracle_lib):
    # Top_2 = {0, 1}, both resident; the first non-candidate (5) is G0 below rank 2
    sST = [0.9, 0.5, 0.1, 0.05, 0.05, 0.5 * (1 - G0), 0.05, 0.05]
    ch, (_, mi, pr, mg) = _refine_step(oracle_lib, sST, (0, 1, 2), R=2)
    assert (mi, pr) == (0, 0) and ch.members() == {0, 1, 2}
    assert mg == pytest.approx(G0, rel=1e-6)


def test_refinement_candidate_order_is_the_margin(oracle_lib):
    # two non-resident candidates 5 and 6 that differ by G0 (their order
    # decides which one meets the lowest resident first)
    sST = [0.9, 0.3, 0.2, 0.01, 0.01, 0.5, 0.5 * (1 - G0), 0.01]
    ch, (_, _, pr, mg) = _refine_step(oracle_lib, sST, (0, 1, 2), R=3)
    assert pr == 2 and ch.members() == {0, 5, 6}
    assert mg == pytest.approx(G0, rel=1e-6)


def test_refinement_argmin_is_the_margin(oracle_lib):
    # candidate 5 replaces the lowest resident 2 (0.1); resident 1 is G0 above it
    sST = [0.9, 0.1 / (1 - G0), 0.1, 0.01, 0.01, 0.7, 0.01, 0.01]
    ch, (_, _, pr, mg) = _refine_step(oracle_lib, sST, (0, 1, 2), R=2)
    assert pr == 1 and ch.members() == {0, 1, 5}
    assert mg == pytest.approx(G0, rel=1e-6)


def test_refinement_strict_test_is_the_margin(oracle_lib):
    # Candidate 5 is G0 above the lowest resident 2: it replaces it (strict >).
    # A candidate's rank gap to its successor is never wider than its gap to
    # a lower resident, so this decision's gap shows up as a rank gap as well;
    # the test checks the margin and the branch taken on both sides of it.
    sST = [0.9, 0.6, 0.3, 0.01, 0.01, 0.3 / (1 - G0), 0.01, 0.01]
    ch, (_, _, pr, mg) = _refine_step(oracle_lib, sST, (0, 1, 2), R=3)
    assert pr == 1 and ch.members() == {0, 1, 5}
    assert mg == pytest.approx(G0, rel=1e-6)
    # G0 below it (R = 4 keeps 5 a candidate): no load, the same margin
    sST[5] = 0.3 * (1 - G0)
    ch, (_, _, pr, mg) = _refine_step(oracle_lib, sST, (0, 1, 2), R=4)
    assert pr == 0 and ch.members() == {0, 1, 2}
    assert mg == pytest.approx(G0, rel=1e-6)


def test_free_slot_fill_takes_no_comparison(oracle_lib):
    # a free slot takes the candidate whatever the residents' scores: the
    # residents 1 and 2 tie exactly, which is no decision here
    sST = [0.9, 0.1, 0.1, 0.01, 0.01, 0.7, 0.01, 0.01]
    ch, (_, _, pr, mg) = _refine_step(oracle_lib, sST, (0, 1, 2), R=2, C=4)
    assert pr == 1 and ch.members() == {0, 1, 2, 5}
    assert mg == pytest.approx(1 - 0.7 / 0.9)     # the rank gap between 0 and 5


def test_exact_ties_exemption(oracle_lib):
    # an exact tie at the Top-K boundary (K = 2): margin 0, unless exact ties
    # are exempt, when the next closest decision (the K/K+1 gap is the tie
    # itself, so nothing else: cold cache) leaves the margin infinite
    N = 8
    p = np.zeros((1, 1, 1, 3, N))
    p[0, 0, 0, 0] = [0.3, 0.2, 0.2, 0.1, 0.1, 0.05, 0.03, 0.02]
    r = oracle_lib.scan(p, K=2, C=3, R=0, margins=True)
    assert r["margins"][0, 0, 0] == 0.0
    assert list(r["topk"][0, 0, 0]) == [0, 1]       # the tie goes to the lower index
    r = oracle_lib.scan(p, K=2, C=3, R=0, margins=True, exact_ties_exempt=True)
    assert r["margins"][0, 0, 0] == np.inf
    assert list(r["topk"][0, 0, 0]) == [0, 1]
    # a close (not exact) pair still counts under the exemption
    p[0, 0, 0, 0, 2] = 0.2 * (1 - G0)
    r = oracle_lib.scan(p, K=2, C=3, R=0, margins=True, exact_ties_exempt=True)
    assert r["margins"][0, 0, 0] == pytest.approx(G0, rel=1e-6)
