"""The formulation of Algorithm 2's refinement that the scan kernels use,
written as a plain model here and checked against the oracle's literal
refinement loop on every cache, capacity, budget and tied score vector of a
small expert count.

The kernels take only the non-resident candidates, in the total order (score
descending, index ascending): the best remaining non-resident c belongs to
A = Top_R exactly when fewer than R experts precede it (its rank); it fills a
free slot, or replaces the cache's last member when strictly higher, and the
first candidate that fails, or whose rank is >= R, ends the pass.  Algorithm 2
walks all of A, residents included; the two must leave the same cache and
count the same proactive loads.
"""
import itertools

import numpy as np
import pytest


def kernel_refine(cache, s, C, R):
    N = len(s)
    key = lambda e: (-s[e], e)                      # position in the total order
    cur = set(cache)
    left = [e for e in range(N) if e not in cur]    # non-residents not yet taken
    pro = 0
    for _ in range(R):
        if not left:
            break
        c = min(left, key=key)
        rank = sum(1 for e in range(N) if key(e) < key(c))
        if rank >= R:
            break
        left.remove(c)
        if len(cur) < C:
            cur.add(c)
            pro += 1
            continue
        v = max(cur, key=key)                       # last member: lowest score, highest index
        if s[c] > s[v]:
            cur.remove(v)
            cur.add(c)
            pro += 1
        else:
            break
    return cur, pro


@pytest.mark.parametrize("N", [4, 5])
def test_rank_formulation_equals_the_literal_loop(oracle_lib, N):
    levels = (0.1, 0.2, 0.3)                        # three values: ties everywhere
    n = 0
    for s in itertools.product(levels, repeat=N):
        s = np.array(s)
        for C in range(1, N + 1):
            for R in range(0, N + 1):
                for size in range(0, C + 1):
                    for cache in itertools.combinations(range(N), size):
                        m = np.zeros(N, np.uint8)
                        m[list(cache)] = 1
                        got, pro, _ = oracle_lib.refine(m, s, C, R)
                        want, pro_k = kernel_refine(set(cache), list(s), C, R)
                        assert set(np.flatnonzero(got)) == want, (s, C, R, cache)
                        assert pro == pro_k, (s, C, R, cache)
                        n += 1
    assert n > 1000
