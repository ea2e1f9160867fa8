"""GPU parity of the comparison policies (crc_cache_scan_policy) against the
oracle's literal scans (oracle.policy_scan) fed the same fp32 probabilities:
bit-exact Top-K trace (rank order), demand misses, proactive loads, final
caches, the policies' integer and float priorities and the counters, for LRU,
LFU, LRFU (lambda = 0, 0.5, 1) and Spatio-only; chunked calls equal one call;
a state keeps the policy of its first call.
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


def probs32(oracle_lib, w, seed, quant=None):
    h, W = S.hidden(w, seed=seed), S.weights(w, seed=seed + 100)
    p = oracle_lib.router_probs(h, W, w.N, H=3)
    if quant:
        p = np.round(p * quant) / quant
    return np.ascontiguousarray(p.astype(np.float32))


def run_gpu(C, w, p32, policy, lam, chunks=None):
    p = C.problem_of(w)
    st = C.State(p)
    T = p32.shape[1]
    tr = C.Trace.alloc(p, T)
    sc = torch.from_numpy(p32).cuda()
    if chunks is None:
        C.cache_scan_policy(p, sc, st, policy, tr, lambda_halves=lam)
    else:
        t0 = 0
        for n in chunks:
            sub = C.Trace.alloc(p, n)
            C.cache_scan_policy(p, sc[:, t0:t0 + n].contiguous(), st, policy, sub, lambda_halves=lam)
            tr.topk[:, t0:t0 + n] = sub.topk
            tr.misses[:, t0:t0 + n] = sub.misses
            tr.proactive[:, t0:t0 + n] = sub.proactive
            t0 += n
    r = st.read(want_caches=True, want_retention=True, want_chain_counters=True)
    r["aux"] = st.read_aux()
    return r, tr


def check(r, tr, o, policy):
    assert r["error"] == 0
    assert np.array_equal(tr.topk.cpu().numpy(), o["topk"])
    assert np.array_equal(tr.misses.cpu().numpy(), o["misses"])
    assert np.array_equal(tr.proactive.cpu().numpy(), o["proactive"])
    assert np.array_equal(r["cache_bits"], o["cache_bits"])
    assert np.array_equal(r["chain_counters"], o["counters"])
    assert np.array_equal(r["aux"], o["aux"])
    if policy in ("lrfu", "spatio_lru"):
        assert np.array_equal(r["retention"].view(np.uint32), o["val"].view(np.uint32))


CASES = [
    ("qwen3", S.QWEN3_30B.with_(B=3, T=80, L=3, d=256), None),
    ("gptoss", S.GPT_OSS_20B.with_(B=4, T=96, L=3, d=256), None),
    ("tiny", S.TINY.with_(T=128), None),
    ("n48", S.QWEN3_30B.with_(B=2, T=64, L=2, d=128, N=48, K=3, C=7, R=2), None),
    ("ties", S.QWEN3_30B.with_(B=2, T=64, L=2, d=128, N=64, K=4, C=9, R=3), 32),
]


@pytest.mark.parametrize("policy", ["lru", "lfu", "lrfu", "spatio_lru"])
@pytest.mark.parametrize("name,w,quant", CASES, ids=[c[0] for c in CASES])
def test_policy_scan_bit_exact(C, oracle_lib, name, w, quant, policy):
    p32 = probs32(oracle_lib, w, seed=3, quant=quant)
    r, tr = run_gpu(C, w, p32, policy, 1)
    o = oracle_lib.policy_scan(p32, w.K, w.C, w.R, policy, lambda2=1)
    check(r, tr, o, policy)
    # Without the rank-order Top-K the kernel takes the Top-K set for 32
    # tokens at a time; untraced, and with misses and proactive loads only,
    # the results are the same.
    p = C.problem_of(w)
    sc = torch.from_numpy(p32).cuda()
    for traced in (False, True):
        st = C.State(p)
        tr2 = C.Trace.alloc(p, w.T, rank_order=False) if traced else None
        C.cache_scan_policy(p, sc, st, policy, tr2, lambda_halves=1)
        r2 = st.read(want_caches=True, want_retention=True, want_chain_counters=True)
        assert r2["error"] == 0
        for k in ("cache_bits", "chain_counters"):
            assert np.array_equal(r2[k], r[k]), (traced, k)
        assert np.array_equal(r2["retention"].view(np.uint32), r["retention"].view(np.uint32))
        assert np.array_equal(st.read_aux(), r["aux"])
        if traced:
            assert torch.equal(tr2.misses, tr.misses) and torch.equal(tr2.proactive, tr.proactive)


@pytest.mark.parametrize("lam", [0, 2])
def test_lrfu_lambdas(C, oracle_lib, lam):
    w = S.QWEN3_30B.with_(B=2, T=120, L=2, d=256)
    p32 = probs32(oracle_lib, w, seed=4)
    r, tr = run_gpu(C, w, p32, "lrfu", lam)
    check(r, tr, oracle_lib.policy_scan(p32, w.K, w.C, w.R, "lrfu", lambda2=lam), "lrfu")


@pytest.mark.parametrize("policy", ["lrfu", "spatio_lru"])
def test_chunked_policy_calls_equal_one_call(C, oracle_lib, policy):
    w = S.QWEN3_30B.with_(B=2, T=100, L=3, d=256)
    p32 = probs32(oracle_lib, w, seed=5)
    r, tr = run_gpu(C, w, p32, policy, 1, chunks=[1, 33, 50, 16])
    check(r, tr, oracle_lib.policy_scan(p32, w.K, w.C, w.R, policy, lambda2=1), policy)


def test_a_state_keeps_its_policy(C, oracle_lib):
    w = S.TINY.with_(T=32)
    p = C.problem_of(w)
    sc = torch.from_numpy(probs32(oracle_lib, w, seed=6)).cuda()
    st = C.State(p)
    C.cache_scan_policy(p, sc, st, "lru")
    assert st.read()["error"] == 0
    C.cache_scan_policy(p, sc, st, "lfu")               # another policy on the same state
    with pytest.raises(C.CrcError):
        st.read()
    st2 = C.State(p)
    C.cache_scan_policy(p, sc, st2, "lru")
    C.cache_scan(p, sc, st2)                            # the method on a policy's state
    with pytest.raises(C.CrcError):
        st2.read()
