"""Pins of the oracle's cache policy: Algorithm 1 (UpdateCache), Algorithm 2
(pre-access refinement + access), the special cases they reduce to, and
hand-traced worked examples."""
import itertools

import numpy as np
import pytest

import crc_synth as S


def order(s, N):
    """Total order of the policy: score descending, expert index ascending."""
    return sorted(range(N), key=lambda e: (-s[e], e))


def update_closed_form(cache, Sset, s, C):
    """Brute force: among all X with S <= X <= C u S and |X| = min(C, |C u S|),
    keep the one whose non-selected part is best under the total order
    (lexicographically smallest sorted key list)."""
    U = cache | Sset
    size = min(C, len(U))
    best = None
    for X in itertools.combinations(sorted(U - Sset), size - len(Sset)):
        k = sorted((-s[e], e) for e in X)
        if best is None or k < best[0]:
            best = (k, set(X) | Sset)
    return best[1]


def refine_closed_form(cache, s, C, R, N):
    """The first min(C, |C u A|) members of C u A, A = Top_R(s), ordered by
    (score desc, resident before candidate, index asc)."""
    A = order(s, N)[:R]
    U = cache | set(A)
    ranked = sorted(U, key=lambda e: (-s[e], 0 if e in cache else 1, e))
    return set(ranked[:min(C, len(U))])


def _mask(sset, N):
    m = np.zeros(N, np.uint8)
    m[list(sset)] = 1
    return m


@pytest.mark.parametrize("dtype", [np.float64, np.float32])
def test_update_cache_brute_force(oracle_lib, dtype):
    N = 5
    scores = list(itertools.product((0.0, 1.0, 2.0), repeat=N))
    n = 0
    for K in (1, 2):
        for C in range(K, 5):
            for csz in range(0, C + 1):
                for cache in itertools.combinations(range(N), csz):
                    cache = set(cache)
                    for Sset in itertools.combinations(range(N), K):
                        Sset = set(Sset)
                        for s in scores[::(7 if dtype == np.float32 else 1)]:
                            got, nd, _ = oracle_lib.update_cache(_mask(cache, N), Sset, s, C, dtype)
                            exp = update_closed_form(cache, Sset, s, C)
                            assert {int(e) for e in np.flatnonzero(got)} == exp, (cache, Sset, s, C)
                            assert nd == len(Sset - cache)
                            n += 1
    assert n > 10000


@pytest.mark.parametrize("dtype", [np.float64, np.float32])
def test_refinement_brute_force(oracle_lib, dtype):
    N = 5
    scores = list(itertools.product((0.0, 1.0, 2.0), repeat=N))
    n = 0
    for C in range(1, 5):
        for R in range(0, N + 1):
            for csz in range(0, C + 1):
                for cache in itertools.combinations(range(N), csz):
                    cache = set(cache)
                    for s in scores[::(5 if dtype == np.float32 else 1)]:
                        got, p, _ = oracle_lib.refine(_mask(cache, N), s, C, R, dtype)
                        got = {int(e) for e in np.flatnonzero(got)}
                        exp = refine_closed_form(cache, s, C, R, N)
                        assert got == exp, (cache, s, C, R)
                        assert p == len(got - cache) and p <= R
                        n += 1
    assert n > 10000


def test_refinement_and_update_random_larger(oracle_lib):
    rng = np.random.default_rng(5)
    for _ in range(3000):
        N = int(rng.integers(6, 40))
        C = int(rng.integers(1, N + 1))
        K = int(rng.integers(1, C + 1))
        R = int(rng.integers(0, N + 1))
        s = rng.integers(0, 6, N).astype(np.float64)      # many ties
        cache = set(rng.choice(N, int(rng.integers(0, C + 1)), replace=False).tolist())
        got, _, _ = oracle_lib.refine(_mask(cache, N), s, C, R)
        assert {int(e) for e in np.flatnonzero(got)} == refine_closed_form(cache, s, C, R, N)
        Sset = set(rng.choice(N, K, replace=False).tolist())
        got, _, _ = oracle_lib.update_cache(_mask(cache, N), Sset, s, C)
        U = cache | Sset
        exp = Sset | set(sorted(U - Sset, key=lambda e: (-s[e], e))[:min(C, len(U)) - K])
        assert {int(e) for e in np.flatnonzero(got)} == exp


# --------------------------------------------------------------------------- #
# hand-traced worked examples (derivations in the comments)
# --------------------------------------------------------------------------- #
def test_worked_example_update_only(oracle_lib):
    """N=5, K=2, C=3, R=0, cold start.
    t0: S={0,1}; cache {} -> 2 misses; free slots -> {0,1}.
    t1: S={2,3} -> 2 misses; s^T=(.35,.15,.45,.35,.70): 2 fills the last slot,
        3 evicts argmin over V={0,1} -> 1 (0.15) -> {0,2,3}.
    t2: S={3,1} (0.40 > 0.35) -> 1 miss (1); s^T=(.2,.45,.15,.5,.7): V={0,2},
        argmin -> 2 (0.15) -> {0,1,3}.
    t3: p^R ties 0.25 at {0,1,2}: TopK by lowest index -> S={0,1}; 0 misses.
    t4: S={3,2} -> 1 miss (2); s^T ties 0.3125 at {0,1}: argmin takes the
        highest index -> evict 1 -> {0,2,3}.   Total: 6 misses, 4 hits."""
    ch = oracle_lib.Chain(5)
    seq = [
        ([.40, .30, .15, .10, .05], [0, 0, 0, 0, 0], [0, 1], 2, {0, 1}),
        ([.05, .10, .40, .30, .15], [.30, .05, .05, .05, .55], [2, 3], 2, {0, 2, 3}),
        ([.10, .35, .05, .40, .10], [.1, .1, .1, .1, .6], [3, 1], 1, {0, 1, 3}),
        ([.25, .25, .25, .125, .125], [0, 0, 0, 0, 0], [0, 1], 0, {0, 1, 3}),
        ([.0625, .0625, .25, .5, .125], [.25, .25, 0, 0, 0], [3, 2], 1, {0, 2, 3}),
    ]
    for t, (pR, pT, topk, mi, cache) in enumerate(seq):
        got_topk, got_mi, got_pr, _ = oracle_lib.step(ch, t, K=2, C=3, R=0, pR=pR, pT=pT)
        assert got_topk == topk and got_mi == mi and got_pr == 0
        assert ch.members() == cache


def test_worked_example_refinement(oracle_lib):
    """N=6, K=1, C=2.
    (a) cache {0,1} full, a^T=(.5,.1,.3,.2,.05,0), p^S=(0,0,.4,.05,.3,.1):
        s^ST=(.5,.1,.7,.25,.35,.1), A=Top_2=[2,0]; 2 replaces argmin{0,1}=1
        (0.7 > 0.1) -> {0,2}, P=1; 0 is resident.  Then S={2}: a hit.
    (b) strict test: s^ST=(.5,.25,.25,0,0,0), R=3, A=[0,1,2]; 2 is not
        strictly above the lowest resident 1 (0.25) -> no load, P=0.
    (c) free slot: cache {0}, s^ST=(.1,.2,.6,.4,0,0), R=3, A=[2,3,1]:
        2 fills the slot; 3 replaces 0 (0.4 > 0.1); 1 loses to 3 (0.2 < 0.4)
        -> {2,3}, P=2."""
    ch = oracle_lib.Chain(6)
    ch.in_cache[[0, 1]] = 1
    ch.count.value = 2
    ch.aT[:] = [.5, .1, .3, .2, .05, 0]
    topk, mi, pr, _ = oracle_lib.step(ch, 1, K=1, C=2, R=2, pR=[.1, .2, .6, .05, .03, .02],
                                      pT=[0] * 6, pS_pred=[0, 0, .4, .05, .3, .1])
    assert (topk, mi, pr) == ([2], 0, 1) and ch.members() == {0, 2}

    got, p, _ = oracle_lib.refine(_mask({0, 1}, 6), [.5, .25, .25, 0, 0, 0], C=2, R=3)
    assert p == 0 and set(np.flatnonzero(got)) == {0, 1}
    got, p, _ = oracle_lib.refine(_mask({0}, 6), [.1, .2, .6, .4, 0, 0], C=2, R=3)
    assert p == 2 and set(np.flatnonzero(got)) == {2, 3}


# --------------------------------------------------------------------------- #
# special cases of the whole scan
# --------------------------------------------------------------------------- #
def _probs(oracle_lib, w, seed=0, const_t=False):
    h = S.hidden(w, seed=seed)
    if const_t:
        h[:] = h[:, :1]
    return oracle_lib.router_probs(h, S.weights(w, seed=seed + 100), w.N)


def test_capacity_equal_k_reduces_to_previous_token_set(oracle_lib):
    w = S.TINY.with_(C=2, K=2, R=0, T=64)
    p = _probs(oracle_lib, w)
    r = oracle_lib.scan(p, w.K, w.C, 0)
    tk = r["topk"]
    for b in range(w.B):
        for l in range(w.L):
            assert r["misses"][b, 0, l] == w.K
            for t in range(1, w.T):
                assert r["misses"][b, t, l] == len(set(tk[b, t, l]) - set(tk[b, t - 1, l]))


def test_capacity_n_counts_distinct_experts(oracle_lib):
    w = S.TINY.with_(C=16, R=0, T=64)
    p = _probs(oracle_lib, w)
    r = oracle_lib.scan(p, w.K, w.C, 0)
    for b in range(w.B):
        for l in range(w.L):
            distinct = set(r["topk"][b, :, l].ravel().tolist())
            assert r["counters"][b, l, 1] == len(distinct)
    # with refinement and C = N nothing is ever evicted: every member entered once
    r = oracle_lib.scan(p, w.K, 16, 3)
    sets = oracle_lib.bits_to_sets(r["cache_bits"], w.N)
    for b in range(w.B):
        for l in range(w.L):
            assert r["counters"][b, l, 1] + r["counters"][b, l, 2] == len(sets[b, l])


def test_constant_hidden_state_misses_only_at_first_token(oracle_lib):
    w = S.TINY.with_(T=32, R=0)
    r = oracle_lib.scan(_probs(oracle_lib, w, const_t=True), w.K, w.C, 0)
    assert np.all(r["misses"][:, 0] == w.K) and np.all(r["misses"][:, 1:] == 0)


def test_r0_is_update_only_and_ignores_spatio(oracle_lib):
    w = S.TINY.with_(T=48, R=0)
    p = _probs(oracle_lib, w)
    q = p.copy()
    q[:, :, :, 2] = np.random.default_rng(0).random(q[:, :, :, 2].shape)
    a, b = oracle_lib.scan(p, w.K, w.C, 0), oracle_lib.scan(q, w.K, w.C, 0)
    for k in ("topk", "misses", "cache_bits", "counters"):
        assert np.array_equal(a[k], b[k])
    assert np.all(a["proactive"] == 0)


def test_refinement_skipped_at_first_token_and_spatio_matters_after(oracle_lib):
    w = S.TINY.with_(T=48, R=2)
    p = _probs(oracle_lib, w)
    r = oracle_lib.scan(p, w.K, w.C, w.R)
    assert np.all(r["proactive"][:, 0] == 0) and r["proactive"].sum() > 0
    q = p.copy()
    q[:, :, :, 2] = q[:, :, :, 2][..., ::-1]
    assert not np.array_equal(oracle_lib.scan(q, w.K, w.C, w.R)["proactive"], r["proactive"])


@pytest.mark.parametrize("R", [0, 1, 3, 16])
def test_invariants(oracle_lib, R):
    w = S.TINY.with_(T=96, R=R)
    r = oracle_lib.scan(_probs(oracle_lib, w, seed=R), w.K, w.C, R)
    c = r["counters"]
    assert np.all(c[..., 0] + c[..., 1] == w.T * w.K)                # hits + misses = T*K
    assert np.all(r["proactive"] <= R)                               # P <= R per access
    assert np.array_equal(c[..., 1], r["misses"].sum(1).astype(np.uint64))
    assert np.array_equal(c[..., 2], r["proactive"].sum(1).astype(np.uint64))
    for cache in oracle_lib.bits_to_sets(r["cache_bits"], w.N).ravel():
        assert len(cache) == w.C                                     # exact capacity once warm
    tk = r["topk"]
    assert all(len(set(row)) == w.K for row in tk.reshape(-1, w.K))


def test_stepwise_replay_equals_scan_and_update_inserts_only_selected(oracle_lib):
    w = S.TINY.with_(T=40, R=2, B=2)
    p = _probs(oracle_lib, w, seed=9)
    r = oracle_lib.scan(p, w.K, w.C, w.R)
    for b in range(w.B):
        chains = [oracle_lib.Chain(w.N) for _ in range(w.L)]
        for t in range(w.T):
            for l in range(w.L):
                pS = None
                if t >= 1:
                    pS = p[b, t, l - 1, 2] if l > 0 else p[b, t - 1, w.L - 1, 2]
                before = chains[l].members()
                A = set()
                if pS is not None and w.R > 0:
                    sST = (p[b, t - 1, l, 0] + p[b, t - 1, l, 1]) + pS
                    A = set(order(sST, w.N)[:w.R])
                tk, mi, pr, _ = oracle_lib.step(chains[l], t, w.K, w.C, w.R,
                                                p[b, t, l, 0], p[b, t, l, 1], pS)
                assert tk == list(r["topk"][b, t, l]) and mi == r["misses"][b, t, l]
                assert pr == r["proactive"][b, t, l]
                # Algorithm 1 inserts only demand-loaded selected experts; every
                # new member comes from S or from the candidates A = Top_R(s^ST).
                assert chains[l].members() - before <= set(tk) | A
        sets = oracle_lib.bits_to_sets(r["cache_bits"][b], w.N)
        assert all(sets[l] == chains[l].members() for l in range(w.L))


def test_fp32_scan_agrees_with_fp64_where_margins_are_wide(oracle_lib):
    w = S.TINY.with_(T=128, R=1)
    p = _probs(oracle_lib, w, seed=4)
    r64 = oracle_lib.scan(p, w.K, w.C, w.R, margins=True)
    r32 = oracle_lib.scan(p.astype(np.float32), w.K, w.C, w.R)
    for b in range(w.B):
        for l in range(w.L):
            bad = np.flatnonzero(r64["margins"][b, :, l] < 1e-3)
            stop = bad[0] if len(bad) else w.T
            assert stop > 0
            assert np.array_equal(r64["topk"][b, :stop, l], r32["topk"][b, :stop, l])
            assert np.array_equal(r64["misses"][b, :stop, l], r32["misses"][b, :stop, l])
            assert np.array_equal(r64["proactive"][b, :stop, l], r32["proactive"][b, :stop, l])


def test_rejects_invalid_sizes(oracle_lib):
    p = np.zeros((1, 1, 1, 3, 8))
    with pytest.raises(ValueError):
        oracle_lib.scan(p, K=3, C=2, R=0)        # C < K
    with pytest.raises(ValueError):
        oracle_lib.scan(p, K=1, C=9, R=0)        # C > N
