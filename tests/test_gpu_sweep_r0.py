"""The update-only capacity sweep at full size: the Qwen3-30B shape with R = 0
(Temporal Router only: no Spatio head, no refinement), B = 256 streams x
T = 2048 tokens, C in {16, 32, 64, 96}.

One hidden-state field (103 GB) and one set of router scores serve every C.
For each C: the fused kernel (one launch) equals the unfused pair on every
chain, bit for bit; the invariants hold on every chain (hits + misses = T.K,
occupancy = C once warm, no proactive load at R = 0); and one whole stream's
scan equals the oracle's literal fp32 scan fed that stream's scores.  Router
rows are checked against the fp64 oracle on sampled units.
"""
import numpy as np
import pytest

import crc_synth as S

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

TOL = 1e-3
W = S.SWEEP_R0


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


@pytest.fixture(scope="module")
def field(C):
    """Hidden states, weights and two-head scores of the sweep, on the device."""
    p = C.problem_of(W)
    Wd = C.synth_weights(W.L, W.N, W.d, seed=0)
    hd, carry = C.synth_hidden(W.B, W.T, W.L, W.d, seed=0, rho_t=W.rho_t, rho_l=W.rho_l)
    del carry
    scores = C.route_scores(p, hd, Wd, heads=2)
    torch.cuda.synchronize()
    yield {"W": Wd, "h": hd, "scores": scores}
    del Wd, hd, scores
    torch.cuda.empty_cache()


def test_sweep_router_rows_vs_oracle(C, oracle_lib, field):
    Wb = host_bits(field["W"])
    hb = field["h"].view(torch.int16)
    rng = np.random.default_rng(1)
    for _ in range(32):
        b, t, l = (int(rng.integers(0, W.B)), int(rng.integers(0, W.T)), int(rng.integers(0, W.L)))
        row = hb[b, t, l].cpu().numpy().view(np.uint16)
        ref = oracle_lib.unit_probs(row, Wb[l], W.N, H=2)
        got = field["scores"][b, t, l, :2].cpu().numpy().astype(np.float64)
        assert (np.abs(got - ref) / np.maximum(np.abs(ref), 1e-30)).max() <= TOL


@pytest.mark.parametrize("cap", W.extra["C_values"])
def test_sweep_capacity_full_size(C, oracle_lib, field, cap):
    w = W.with_(C=cap)
    p = C.problem_of(w)

    # fused route-and-cache, as the benchmark issues it
    ws = torch.empty(C.crc_fused_workspace_bytes(p), dtype=torch.uint8, device="cuda")
    stf = C.State(p)
    C.crc_profile_begin()
    C.route_and_cache(p, field["h"], field["W"], stf, None, workspace=ws)
    assert C.crc_profile_end()["fused"]["launches"] == 1
    fz = stf.read(want_caches=True, want_retention=True, want_chain_counters=True)
    del ws
    assert fz["error"] == 0 and fz["tokens"] == w.T

    # the pair: scan of the precomputed scores
    stp = C.State(p)
    C.cache_scan(p, field["scores"], stp)
    pr = stp.read(want_caches=True, want_retention=True, want_chain_counters=True)
    assert pr["error"] == 0
    assert np.array_equal(fz["cache_bits"], pr["cache_bits"])
    assert np.array_equal(fz["chain_counters"], pr["chain_counters"])
    assert np.array_equal(fz["retention"].view(np.uint32), pr["retention"].view(np.uint32))

    # invariants on every chain
    cc = fz["chain_counters"]
    assert np.all(cc[..., 0] + cc[..., 1] == w.T * w.K)
    assert np.all(cc[..., 2] == 0)                       # R = 0: no proactive load
    pop = np.vectorize(lambda x: bin(int(x)).count("1"))(fz["cache_bits"]).sum(-1)
    assert np.all(pop == cap)

    # one whole stream: the oracle's literal fp32 scan on the same scores
    b = (cap * 7) % w.B
    s32 = field["scores"][b].cpu().numpy()[None]
    o = oracle_lib.scan(s32, w.K, w.C, w.R, trace=False)
    assert np.array_equal(fz["cache_bits"][b], o["cache_bits"][0])
    assert np.array_equal(fz["retention"][b].view(np.uint32), o["aT"][0].view(np.uint32))
    assert np.array_equal(fz["chain_counters"][b], o["counters"][0])
