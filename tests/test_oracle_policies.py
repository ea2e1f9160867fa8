"""The oracle's comparison policies (the paper's LRU / LFU / LRFU cache-update
baselines and the Spatio-only ablation), pinned to things other than
themselves:

* LRU and LFU against textbook simulators written here from scratch: an
  OrderedDict recency list and an in-cache frequency table (victims outside
  the access's Top-K set, ties to the highest expert index);
* LRFU with lambda = 0 is LFU (F = 1, so the CRF is the access count);
* LRFU(0.5) on hand-worked traces where it disagrees with LRU and with LFU;
* Spatio-only with R = 0 is LRU;
* invariants on random inputs for every policy.
"""
from collections import OrderedDict

import numpy as np
import pytest

POLICIES = ("lru", "lfu", "lrfu", "spatio_lru")


def _probs(rng, B, T, L, N, ties=False):
    p = rng.random((B, T, L, 3, N)).astype(np.float32)
    if ties:
        p = np.round(p * 8) / 8
    return p.astype(np.float32)


def _sets(res, b, l):
    return [set(int(e) for e in row) for row in res["topk"][b, :, l]]


def textbook_lru(sets, C):
    cache, misses = OrderedDict(), []      # least recently used first
    for S in sets:
        m = 0
        for e in sorted(S):
            if e in cache:
                continue
            m += 1
            if len(cache) >= C:
                del cache[next(v for v in cache if v not in S)]
            cache[e] = None
        for e in sorted(S, reverse=True):   # same-token uses: highest index least recent
            cache.move_to_end(e)
        misses.append(m)
    return set(cache), misses


def textbook_lfu(sets, C):
    count, misses = {}, []
    for S in sets:
        m = 0
        for e in sorted(S):
            if e in count:
                continue
            m += 1
            if len(count) >= C:
                victim = min((v for v in count if v not in S), key=lambda v: (count[v], -v))
                del count[victim]
            count[e] = 0
        for e in S:
            count[e] += 1
        misses.append(m)
    return set(count), misses


@pytest.mark.parametrize("ties", [False, True])
@pytest.mark.parametrize("N,K,C", [(16, 2, 4), (16, 4, 7), (32, 3, 3), (8, 1, 5)])
def test_lru_and_lfu_match_textbook_simulators(oracle_lib, N, K, C, ties):
    rng = np.random.default_rng(N * 100 + K * 10 + C + ties)
    p = _probs(rng, 3, 60, 2, N, ties)
    for pol, sim in (("lru", textbook_lru), ("lfu", textbook_lfu)):
        r = oracle_lib.policy_scan(p, K, C, 0, pol)
        for b in range(3):
            for l in range(2):
                cache, misses = sim(_sets(r, b, l), C)
                got = {e for e in range(N) if (int(r["cache_bits"][b, l, e // 32]) >> (e % 32)) & 1}
                assert got == cache, (pol, b, l)
                assert list(r["misses"][b, :, l]) == misses, (pol, b, l)


def test_lrfu_with_lambda_zero_is_lfu(oracle_lib):
    rng = np.random.default_rng(11)
    p = _probs(rng, 4, 80, 3, 16, ties=True)
    a = oracle_lib.policy_scan(p, 2, 5, 0, "lrfu", lambda2=0)
    b = oracle_lib.policy_scan(p, 2, 5, 0, "lfu")
    for k in ("cache_bits", "counters", "topk", "misses"):
        assert np.array_equal(a[k], b[k]), k
    # for every cached expert the CRF equals its access count since insertion
    N = p.shape[-1]
    e = np.arange(N)
    resident = ((b["cache_bits"][..., e // 32] >> (e % 32)) & 1).astype(bool)
    assert np.array_equal(a["val"][resident], b["aux"][resident].astype(np.float32))


def _one_hot_trace(choices, N):
    """Native Top-1 choices as probabilities: the chosen expert gets 0.7."""
    p = np.full((1, len(choices), 1, 3, N), 0.1, np.float32)
    for t, e in enumerate(choices):
        p[0, t, 0, 0, e] = 0.7
    return p


def _final(res, N):
    return {e for e in range(N) if (int(res["cache_bits"][0, 0, e // 32]) >> (e % 32)) & 1}


def test_lrfu_worked_examples(oracle_lib):
    N = 4
    # 0, 0, 1, then 2 into a full cache {0, 1}:
    # CRF_0 = 1 + 2^-0.5 at t1, decayed by 2^-1 to t3 -> 0.854; CRF_1 = 1 at t2 -> 0.707
    p = _one_hot_trace([0, 0, 1, 2], N)
    assert _final(oracle_lib.policy_scan(p, 1, 2, 0, "lrfu"), N) == {0, 2}   # keeps the frequent one
    assert _final(oracle_lib.policy_scan(p, 1, 2, 0, "lru"), N) == {1, 2}    # keeps the recent one
    # 0, 0, 0, 1, 1, then 2: counts 3 vs 2, but CRF_0 = 2.207 * 2^-1.5 = 0.780 and
    # CRF_1 = 1.707 * 2^-0.5 = 1.207 at t5
    p = _one_hot_trace([0, 0, 0, 1, 1, 2], N)
    assert _final(oracle_lib.policy_scan(p, 1, 2, 0, "lrfu"), N) == {1, 2}   # recency wins
    assert _final(oracle_lib.policy_scan(p, 1, 2, 0, "lfu"), N) == {0, 2}    # frequency wins


def test_spatio_only_without_candidates_is_lru(oracle_lib):
    rng = np.random.default_rng(12)
    p = _probs(rng, 3, 70, 4, 32)
    a = oracle_lib.policy_scan(p, 4, 9, 0, "spatio_lru")
    b = oracle_lib.policy_scan(p, 4, 9, 0, "lru")
    for k in ("cache_bits", "counters", "topk", "misses", "aux"):
        assert np.array_equal(a[k], b[k]), k


@pytest.mark.parametrize("pol", POLICIES)
def test_policy_invariants(oracle_lib, pol):
    rng = np.random.default_rng(13)
    B, T, L, N, K, C, R = 3, 90, 3, 32, 4, 9, 3
    r = oracle_lib.policy_scan(_probs(rng, B, T, L, N), K, C, R, pol)
    cc = r["counters"]
    assert np.all(cc[..., 0] + cc[..., 1] == T * K)
    pop = np.vectorize(lambda x: bin(int(x)).count("1"))(r["cache_bits"]).sum(-1)
    assert np.all(pop == C)                                   # warm after 90 tokens
    if pol == "spatio_lru":
        assert int(r["proactive"].max()) <= R and int(cc[..., 2].sum()) > 0
    else:
        assert int(cc[..., 2].sum()) == 0 and int(r["proactive"].max()) == 0
    assert int(r["misses"].max()) <= K                        # demand loads per access
