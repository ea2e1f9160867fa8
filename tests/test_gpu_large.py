"""The large configuration at full size, streamed: the Qwen3-235B-A22B shape
(L = 94, N = 128, K = 8, d = 4096, C = 32), B = 512 streams x T = 4096
tokens, R in {2, 8}.  Its hidden states (1.61 TB) never exist at once: the
device generator writes 128-token chunks (the AR(1) field continues across
chunks through its carry), and each chunk goes through both paths on
persistent states, exactly as successive calls of a decode loop would:

* the fused route-and-cache kernel (no trace, fused workspace), and
* route_scores + cache_scan (the pair).

Checked: the two final states are identical on every chain (caches,
retention, counters); the invariants hold on every chain; one whole stream
(all 4096 tokens x 94 layers) equals the oracle's literal fp32 scan fed that
stream's scores; sampled router rows match the fp64 oracle.
"""
import numpy as np
import pytest

import crc_synth as S

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

TOL = 1e-3
CHUNK = 128


@pytest.fixture(scope="module")
def C():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2609_04895_gb300 import build
    build.build()
    from paper_2609_04895_gb300 import crc
    crc.load()
    return crc


def host_bits(t) -> np.ndarray:
    return t.view(torch.int16).cpu().numpy().view(np.uint16)


@pytest.mark.parametrize("R", S.LARGE.extra["R_values"])
def test_large_streamed_full_size(C, oracle_lib, R):
    w = S.LARGE.with_(R=R)
    p = C.problem_of(w)
    Wd = C.synth_weights(w.L, w.N, w.d, seed=0)
    Wb = host_bits(Wd)
    hbuf = torch.empty((w.B, CHUNK, w.L, w.d), dtype=torch.bfloat16, device="cuda")
    carry = torch.zeros((w.B, w.L, w.d), dtype=torch.float32, device="cuda")
    scores = torch.empty((w.B, CHUNK, w.L, 3, w.N), dtype=torch.float32, device="cuda")
    ws = torch.empty(C.crc_fused_workspace_bytes(p), dtype=torch.uint8, device="cuda")
    stf, stp = C.State(p), C.State(p)
    b_s = (R * 97) % w.B                     # the stream checked against the oracle
    s_host = np.empty((w.T, w.L, 3, w.N), np.float32)
    rng = np.random.default_rng(R)
    worst = 0.0
    try:
        C.crc_profile_begin()
        for c in range(w.T // CHUNK):
            t0 = c * CHUNK
            C.synth_hidden(w.B, CHUNK, w.L, w.d, seed=0, rho_t=w.rho_t, rho_l=w.rho_l, t0=t0,
                           carry=carry, out=hbuf)
            C.route_and_cache(p, hbuf, Wd, stf, None, workspace=ws)
            C.route_scores(p, hbuf, Wd, heads=3, out=scores)
            C.cache_scan(p, scores, stp)
            s_host[t0:t0 + CHUNK] = scores[b_s].cpu().numpy()
            # two sampled router rows per chunk vs the fp64 oracle
            for _ in range(2):
                b, t, l = (int(rng.integers(0, w.B)), int(rng.integers(0, CHUNK)),
                           int(rng.integers(0, w.L)))
                row = hbuf[b, t, l].view(torch.int16).cpu().numpy().view(np.uint16)
                ref = oracle_lib.unit_probs(row, Wb[l], w.N, H=3)
                got = scores[b, t, l].cpu().numpy().astype(np.float64)
                worst = max(worst, float((np.abs(got - ref) /
                                          np.maximum(np.abs(ref), 1e-30)).max()))
        prof = C.crc_profile_end()
    finally:
        del hbuf, scores, ws, carry
        torch.cuda.empty_cache()
    assert worst <= TOL
    assert prof["fused"]["launches"] == w.T // CHUNK

    fz = stf.read(want_caches=True, want_retention=True, want_chain_counters=True)
    pr = stp.read(want_caches=True, want_retention=True, want_chain_counters=True)
    assert fz["error"] == 0 and pr["error"] == 0
    assert fz["tokens"] == w.T and pr["tokens"] == w.T
    assert np.array_equal(fz["cache_bits"], pr["cache_bits"])
    assert np.array_equal(fz["chain_counters"], pr["chain_counters"])
    assert np.array_equal(fz["retention"].view(np.uint32), pr["retention"].view(np.uint32))

    cc = fz["chain_counters"]
    assert np.all(cc[..., 0] + cc[..., 1] == w.T * w.K)
    assert int(cc[..., 2].max()) <= w.T * w.R
    pop = np.vectorize(lambda x: bin(int(x)).count("1"))(fz["cache_bits"]).sum(-1)
    assert np.all(pop == w.C)
    assert fz["traffic_bytes"] == (fz["misses"] + fz["proactive"]) * w.expert_bytes

    o = oracle_lib.scan(s_host[None], w.K, w.C, w.R, trace=False)
    assert np.array_equal(fz["cache_bits"][b_s], o["cache_bits"][0])
    assert np.array_equal(fz["retention"][b_s].view(np.uint32), o["aT"][0].view(np.uint32))
    assert np.array_equal(fz["chain_counters"][b_s], o["counters"][0])
