"""The expert-transfer planner (crc_transfer_plan, host only), pinned to:

* a hand-worked sequence of cache sets with the exact copies and slots;
* cache trajectories of the oracle (Algorithm 2 refinement, then Algorithm 1
  update, per access): the plan holds exactly the oracle's proactive loads P
  and demand misses D, every slot holds at most one expert, the slot map
  always equals the cache set, and planning token by token equals planning
  the whole sequence at once;
* argument checks (no GPU is used).
"""
import numpy as np
import pytest

import crc_synth as S


@pytest.fixture(scope="module")
def C():
    from paper_2609_04895_gb300 import build
    build.build()
    from paper_2609_04895_gb300 import crc
    crc.load()
    return crc


def words(sets, N):
    nw = (N + 31) // 32
    out = np.zeros(nw, np.uint32)
    for e in sets:
        out[e // 32] |= np.uint32(1 << (e % 32))
    return out


def test_hand_worked_sequence(C):
    p = C.problem(L=1, N=8, K=2, d=16, C=3, R=1, B=1, expert_bytes=64)
    #          mid (after refinement)   after (after UpdateCache)
    steps = [({},                    {0, 1}),        # t0: demand 0, 1 into slots 0, 1
             ({0, 1, 5},             {0, 1, 5}),     # t1: proactive 5 into slot 2
             ({0, 1, 6},             {0, 3, 6}),     # t2: 6 replaces 5; demand 3 replaces 1
             ({0, 3, 6},             {2, 4, 6})]     # t3: demand 2, 4 replace 0, 3
    mid = np.stack([words(m, 8) for m, _ in steps])[:, None, :]
    aft = np.stack([words(a, 8) for _, a in steps])[:, None, :]
    plan, se = C.transfer_plan(p, mid, aft)
    got = [(int(x["t"]), int(x["expert"]), int(x["slot"]), int(x["evicted"]), int(x["proactive"]))
           for x in plan]
    assert got == [(0, 0, 0, -1, 0), (0, 1, 1, -1, 0),
                   (1, 5, 2, -1, 1),
                   (2, 6, 2, 5, 1), (2, 3, 1, 1, 0),
                   (3, 2, 0, 0, 0), (3, 4, 1, 3, 0)]
    assert sorted(se[0].tolist()) == [2, 4, 6] and se[0].tolist() == [2, 4, 6]


def oracle_trajectory(oracle_lib, probs, K, Ccap, R):
    """Per-access cache sets of one stream from the oracle: after Algorithm 2
    and after Algorithm 1, with the oracle's own P and D."""
    T, L, _, N = probs.shape
    chains = [oracle_lib.Chain(N) for _ in range(L)]
    nw = (N + 31) // 32
    mid = np.zeros((T, L, nw), np.uint32)
    aft = np.zeros((T, L, nw), np.uint32)
    P = D = 0
    for t in range(T):
        for l in range(L):
            ch = chains[l]
            pS = probs[t, l - 1, 2] if l > 0 else (probs[t - 1, L - 1, 2] if t > 0 else None)
            if R > 0 and t >= 1:
                m, _, _ = oracle_lib.refine(ch.in_cache, ch.aT + pS, Ccap, R)
            else:
                m = ch.in_cache.copy()
            _, mi, pr, _ = oracle_lib.step(ch, t, K, Ccap, R, probs[t, l, 0], probs[t, l, 1],
                                           pS if (R > 0 and t >= 1) else None)
            mid[t, l] = words(np.flatnonzero(m), N)
            aft[t, l] = words(ch.members(), N)
            P += pr
            D += mi
    return mid, aft, P, D, [ch.members() for ch in chains]


@pytest.mark.parametrize("N,K,Ccap,R", [(16, 2, 4, 1), (32, 4, 8, 2), (64, 4, 9, 3)])
def test_plan_follows_oracle_trajectories(C, oracle_lib, N, K, Ccap, R):
    T, L = 40, 3
    probs = S.distributions(1, T, L, N, seed=N + K)[0].astype(np.float64)
    mid, aft, P, D, final = oracle_trajectory(oracle_lib, probs, K, Ccap, R)
    p = C.problem(L=L, N=N, K=K, d=16, C=Ccap, R=R, B=1, expert_bytes=256)
    plan, se = C.transfer_plan(p, mid, aft)
    assert int((plan["proactive"] == 1).sum()) == P
    assert int((plan["proactive"] == 0).sum()) == D
    for l in range(L):
        slots = [e for e in se[l].tolist() if e >= 0]
        assert len(slots) == len(set(slots)) and set(slots) == final[l]
    # replay the plan on a slot map: every copy lands in a slot that is free or
    # freed by the expert it names, and the map equals the cache after each access
    smap = np.full((L, Ccap), -1)
    i = 0
    for t in range(T):
        for l in range(L):
            for phase, target in ((1, mid[t, l]), (0, aft[t, l])):
                keep = {e for e in range(N) if (int(target[e // 32]) >> (e % 32)) & 1}
                for s in range(Ccap):
                    if smap[l, s] >= 0 and smap[l, s] not in keep:
                        smap[l, s] = -1
                while i < len(plan) and plan[i]["t"] == t and plan[i]["l"] == l and \
                        plan[i]["proactive"] == phase:
                    x = plan[i]
                    assert smap[l, x["slot"]] == -1
                    smap[l, x["slot"]] = x["expert"]
                    i += 1
                assert {e for e in smap[l] if e >= 0} == keep
    assert i == len(plan)
    # token by token gives the same copies
    se2 = np.full((L, Ccap), -1, np.int32)
    parts = []
    for t in range(T):
        start = aft[t - 1] if t > 0 else None
        part, se2 = C.transfer_plan(p, mid[t:t + 1], aft[t:t + 1], slot_expert=se2, start=start)
        part["t"] += t
        parts.append(part)
    whole = np.concatenate(parts)
    assert np.array_equal(whole, plan)


def test_argument_checks(C):
    p = C.problem(L=1, N=8, K=2, d=16, C=2, R=1, B=1, expert_bytes=64)
    three = np.stack([words({0, 1, 2}, 8)])[:, None, :]
    with pytest.raises(C.CrcError):                 # three members in a 2-slot cache
        C.transfer_plan(p, three, three)
    ok = np.stack([words({0, 1}, 8)])[:, None, :]
    with pytest.raises(C.CrcError):                 # start set disagrees with the slot map
        C.transfer_plan(p, ok, ok, slot_expert=np.array([[0, -1]]), start=words({3}, 8)[None, :])
    with pytest.raises(C.CrcError):                 # an expert in two slots
        C.transfer_plan(p, ok, ok, slot_expert=np.array([[1, 1]]))
    lib = C.load()
    assert lib.crc_transfer_replay(None, None, 0, None, 1, None, None) == C.CRC_EINVAL
