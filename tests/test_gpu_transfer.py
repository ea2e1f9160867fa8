"""GPU side of the expert transfers: the scan's per-access cache sets (after
Algorithm 2 and after Algorithm 1) bit-exact against the oracle's fp32
trajectory; the same sets through crc_route_and_cache; and a replay of one
stream's plan with distinct expert images: every slot ends up holding the
bytes of the expert the plan put there, and the bytes moved equal
(misses + proactive loads) x expert_bytes of that stream's counters.
"""
import numpy as np
import pytest

import crc_synth as S

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def C():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2609_04895_gb300 import build
    build.build()
    from paper_2609_04895_gb300 import crc
    crc.load()
    return crc


def words(sets, N):
    out = np.zeros((N + 31) // 32, np.uint32)
    for e in sets:
        out[e // 32] |= np.uint32(1 << (e % 32))
    return out


def oracle_masks(oracle_lib, probs, K, Ccap, R):
    """fp32 oracle trajectory of every stream: [B][T][L][NW] after the
    refinement and after UpdateCache."""
    B, T, L, _, N = probs.shape
    nw = (N + 31) // 32
    mid = np.zeros((B, T, L, nw), np.uint32)
    aft = np.zeros((B, T, L, nw), np.uint32)
    for b in range(B):
        chains = [oracle_lib.Chain(N, np.float32) for _ in range(L)]
        for t in range(T):
            for l in range(L):
                ch = chains[l]
                pS = probs[b, t, l - 1, 2] if l > 0 else (probs[b, t - 1, L - 1, 2] if t else None)
                use_s = R > 0 and t >= 1
                if use_s:
                    m, _, _ = oracle_lib.refine(ch.in_cache, (ch.aT + pS).astype(np.float32),
                                                Ccap, R, dtype=np.float32)
                else:
                    m = ch.in_cache.copy()
                oracle_lib.step(ch, t, K, Ccap, R, probs[b, t, l, 0], probs[b, t, l, 1],
                                pS if use_s else None)
                mid[b, t, l] = words(np.flatnonzero(m), N)
                aft[b, t, l] = words(ch.members(), N)
    return mid, aft


CASES = [("qwen3", S.QWEN3_30B.with_(B=2, T=48, L=3, d=128)),
         ("gptoss", S.GPT_OSS_20B.with_(B=2, T=48, L=3, d=128)),
         ("n48", S.QWEN3_30B.with_(B=2, T=40, L=2, d=128, N=48, K=3, C=7, R=2))]


@pytest.mark.parametrize("name,w", CASES, ids=[c[0] for c in CASES])
def test_cache_trace_matches_oracle(C, oracle_lib, name, w):
    probs = S.distributions(w.B, w.T, w.L, w.N, seed=21)
    p = C.problem_of(w)
    st = C.State(p)
    tr = C.Trace.alloc(p, w.T, caches=True)
    C.cache_scan(p, torch.from_numpy(probs).cuda(), st, tr)
    assert st.read()["error"] == 0
    mid, aft = oracle_masks(oracle_lib, probs, w.K, w.C, w.R)
    assert np.array_equal(tr.cache_mid.cpu().numpy().view(np.uint32), mid)
    assert np.array_equal(tr.cache_after.cpu().numpy().view(np.uint32), aft)
    # proactive loads and misses of the trace agree with the masks
    pro = tr.proactive.cpu().numpy().astype(np.int64)
    miss = tr.misses.cpu().numpy().astype(np.int64)
    pc = np.vectorize(lambda x: bin(int(x)).count("1"))
    before = np.concatenate([np.zeros_like(aft[:, :1]), aft[:, :-1]], axis=1)
    assert np.array_equal(pc(mid & ~before).sum(-1), pro)
    assert np.array_equal(pc(aft & ~mid).sum(-1), miss)


def test_route_and_cache_writes_the_same_trace(C):
    w = S.QWEN3_30B.with_(B=2, T=40, L=3, d=256)
    p = C.problem_of(w)
    Wd = C.synth_weights(w.L, w.N, w.d, seed=3)
    hd, _ = C.synth_hidden(w.B, w.T, w.L, w.d, seed=4)
    scores = C.route_scores(p, hd, Wd)
    st1, st2 = C.State(p), C.State(p)
    t1, t2 = C.Trace.alloc(p, w.T, caches=True), C.Trace.alloc(p, w.T, caches=True)
    C.cache_scan(p, scores, st1, t1)
    C.route_and_cache(p, hd, Wd, st2, t2)
    assert st1.read()["error"] == 0 and st2.read()["error"] == 0
    assert torch.equal(t1.cache_mid, t2.cache_mid) and torch.equal(t1.cache_after, t2.cache_after)


def test_replay_moves_each_planned_expert(C):
    w = S.QWEN3_30B.with_(B=3, T=64, L=4, d=128, N=32, K=4, C=8, R=2, expert_bytes=4096)
    probs = S.distributions(w.B, w.T, w.L, w.N, seed=22)
    p = C.problem_of(w)
    st = C.State(p)
    tr = C.Trace.alloc(p, w.T, caches=True)
    C.cache_scan(p, torch.from_numpy(probs).cuda(), st, tr)
    r = st.read(want_caches=True, want_chain_counters=True)
    assert r["error"] == 0
    b = 1
    mid = tr.cache_mid[b].cpu().numpy()
    aft = tr.cache_after[b].cpu().numpy()
    plan, se = C.transfer_plan(p, mid, aft)
    counters = r["chain_counters"].reshape(w.B, w.L, 3)[b]
    assert len(plan) == int(counters[:, 1].sum() + counters[:, 2].sum())     # D + P
    eb = w.expert_bytes
    # distinct images: byte i of expert (l, e) = (l * 37 + e * 11 + i) mod 251
    img = (np.arange(w.L)[:, None, None] * 37 + np.arange(w.N)[None, :, None] * 11
           + np.arange(eb)[None, None, :]) % 251
    pool = torch.from_numpy(img.astype(np.uint8).reshape(-1)).pin_memory()
    slots = torch.zeros((w.L, w.C, eb), dtype=torch.uint8, device="cuda")
    C.transfer_replay(p, plan, pool, slots)
    torch.cuda.synchronize()
    got = slots.cpu().numpy()
    for l in range(w.L):
        for s in range(w.C):
            e = int(se[l, s])
            if e >= 0:
                assert np.array_equal(got[l, s], img[l, e].astype(np.uint8)), (l, s, e)
    final = {(l, int(e)) for l in range(w.L) for e in se[l] if e >= 0}
    bits = r["cache_bits"].reshape(w.B, w.L, -1)[b]
    assert final == {(l, e) for l in range(w.L) for e in range(w.N)
                     if (int(bits[l, e // 32]) >> (e % 32)) & 1}
