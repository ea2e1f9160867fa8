"""End to end against the fp64 oracle at full size, on margin-certified inputs.

The GPU decides in fp32, the oracle in fp64; their decisions agree wherever
each decision's two scores are at least 1e-3 apart (relative), since the
router heads are within 2.5e-4 of the fp64 values.  ``oracle.certify`` walks
sampled streams of the Qwen3-30B- and GPT-OSS-20B-shaped workloads unit by
unit in causal order and redraws the innovation of any unit whose draw would
put a decision closer than that (its own access, or the refinement of the
next unit, whose causal predecessor it is).  The device generator then
writes the whole workload with that re-draw table, the benchmark's fused
kernel runs over it, and on the sampled streams every per-access decision --
the native Top-K set (Sec. 2), the demand misses and the proactive loads of
Algorithm 2, the final caches after Algorithm 1 and the counters -- must
equal the fp64 oracle's, over all T tokens of every layer.  Cases: Tiny (all
four streams), the Qwen3-30B and GPT-OSS-20B shapes (eight streams each) and
the update-only sweep at C = 16 and C = 96 (four of its 256 streams each).
"""
import numpy as np
import pytest

import crc_synth as S

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

TOL = 1e-3


@pytest.fixture(scope="module")
def C():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2609_04895_gb300 import build
    build.build()
    from paper_2609_04895_gb300 import crc
    crc.load()
    return crc


def _sets(topk: np.ndarray, N: int) -> np.ndarray:
    """[..., K] expert indices -> [..., NW] uint32 bitmasks."""
    NW = (N + 31) // 32
    out = np.zeros(topk.shape[:-1] + (NW,), np.uint32)
    for k in range(topk.shape[-1]):
        e = topk[..., k].astype(np.int64)
        np.bitwise_or.at(out.reshape(-1, NW), (np.arange(e.size), (e // 32).ravel()),
                         (np.uint32(1) << (e % 32).astype(np.uint32)).ravel())
    return out


CASES = [
    (S.TINY, (0, 1, 2, 3)),                                          # every stream
    (S.QWEN3_30B, (0, 9, 18, 27, 36, 45, 54, 63)),
    (S.GPT_OSS_20B, (0, 17, 34, 51, 68, 85, 102, 127)),
    # the update-only sweep (R = 0) at its smallest and largest capacity
    (S.SWEEP_R0.with_(C=16), (0, 85, 170, 255)),
    (S.SWEEP_R0.with_(C=96), (0, 85, 170, 255)),
]


@pytest.mark.parametrize("w,streams", CASES, ids=[f"{c[0].name}-C{c[0].C}" for c in CASES])
def test_certified_streams_equal_fp64_oracle(C, oracle_lib, w, streams):
    from oracle import certify
    W = S.weights(w, seed=0)
    cert = certify.certified_streams(w, W, seed=0, streams=streams, tol=TOL)
    covered = float(cert["certified"].mean())
    print(f"\n{w.name}: {len(streams)} streams x {w.T} tokens x {w.L} layers, "
          f"{int(cert['redraws'].sum())} redraws, certified {covered:.5f}")
    assert covered >= 0.999

    # the whole workload from the device generator with the re-draw table
    att = np.zeros((w.B, w.T, w.L), np.uint8)
    att[list(streams)] = cert["attempts"]
    att_d = torch.from_numpy(att).cuda()
    Wd = C.synth_weights(w.L, w.N, w.d, seed=0)
    hd, _ = C.synth_hidden(w.B, w.T, w.L, w.d, seed=0, rho_t=w.rho_t, rho_l=w.rho_l,
                           attempts=att_d)
    del att_d
    for i, b in enumerate(streams):
        ref = torch.from_numpy(cert["hidden"][i].view(np.int16)).cuda()
        assert torch.equal(hd[b].view(torch.int16), ref), b
        del ref

    p = C.problem_of(w)
    ws = torch.empty(C.crc_fused_workspace_bytes(p), dtype=torch.uint8, device="cuda")
    # the benchmark's call: one fused kernel, no trace
    st = C.State(p)
    C.crc_profile_begin()
    C.route_and_cache(p, hd, Wd, st, None, workspace=ws)
    assert C.crc_profile_end()["fused"]["launches"] == 1
    fz = st.read(want_caches=True, want_retention=True, want_chain_counters=True)
    assert fz["error"] == 0 and fz["tokens"] == w.T
    # the same fused kernel writing its per-access trace
    st2 = C.State(p)
    tr = C.Trace.alloc(p, w.T, rank_order=False, topk_set=True)
    C.crc_profile_begin()
    C.route_and_cache(p, hd, Wd, st2, tr, workspace=ws)
    assert C.crc_profile_end()["fused"]["launches"] == 1
    tz = st2.read(want_caches=True, want_retention=True, want_chain_counters=True)
    for k in ("cache_bits", "chain_counters"):
        assert np.array_equal(tz[k], fz[k]), k
    assert np.array_equal(tz["retention"].view(np.uint32), fz["retention"].view(np.uint32))

    idx = list(streams)
    g_set = tr.topk_set[idx].cpu().numpy().view(np.uint32)
    g_mis = tr.misses[idx].cpu().numpy()
    g_pro = tr.proactive[idx].cpu().numpy()
    o_set = _sets(cert["topk"], w.N)
    n_full = 0
    for i in range(len(idx)):
        for l in range(w.L):
            bad = np.flatnonzero(~cert["certified"][i, :, l])
            stop = int(bad[0]) if len(bad) else w.T
            sl = slice(0, stop)
            assert np.array_equal(g_set[i, sl, l], o_set[i, sl, l]), (idx[i], l)
            assert np.array_equal(g_mis[i, sl, l], cert["misses"][i, sl, l]), (idx[i], l)
            assert np.array_equal(g_pro[i, sl, l], cert["proactive"][i, sl, l]), (idx[i], l)
            if stop == w.T:
                n_full += 1
                b = idx[i]
                assert np.array_equal(fz["cache_bits"][b, l], cert["cache_bits"][i, l])
                assert np.array_equal(fz["chain_counters"][b, l], cert["counters"][i, l])
                ref = cert["aT"][i, l]
                err = np.abs(fz["retention"][b, l].astype(np.float64) - ref) / ref
                assert err.max() <= TOL
    assert n_full >= 0.95 * len(idx) * w.L
    # traffic of the fully certified chains = (misses + proactive) x expert bytes
    if n_full == len(idx) * w.L:
        cc = fz["chain_counters"][idx]
        traffic = (int(cc[..., 1].sum()) + int(cc[..., 2].sum())) * w.expert_bytes
        oc = cert["counters"]
        assert traffic == (int(oc[..., 1].sum()) + int(oc[..., 2].sum())) * w.expert_bytes


@pytest.mark.parametrize("R", S.LARGE.extra["R_values"])
def test_large_certified_prefix(C, oracle_lib, R):
    """The large shape (L = 94, d = 4096, B = 512) streamed in 128-token
    chunks as the benchmark runs it: the first 256 tokens of two sampled
    streams are drawn margin-certified (a whole stream is a quarter of an hour
    of fp64 oracle work), the device generator writes both chunks with that
    re-draw table, and the fused kernel's per-access decisions and the chain
    states after 256 tokens equal the fp64 oracle's."""
    from oracle import certify
    TC, CH = 256, 128
    w = S.LARGE.with_(R=R)
    wc = w.with_(T=TC)
    streams = ((R * 97) % w.B, (R * 97 + 256) % w.B)
    Wd = C.synth_weights(w.L, w.N, w.d, seed=0)
    Wb = Wd.view(torch.int16).cpu().numpy().view(np.uint16)
    cert = certify.certified_streams(wc, Wb, seed=0, streams=streams, tol=TOL)
    print(f"\nlarge R={R}: {len(streams)} streams x {TC} tokens x {w.L} layers, "
          f"{int(cert['redraws'].sum())} redraws, certified {float(cert['certified'].mean()):.5f}")
    assert cert["certified"].mean() >= 0.999
    p = C.problem_of(w)
    hbuf = torch.empty((w.B, CH, w.L, w.d), dtype=torch.bfloat16, device="cuda")
    carry = torch.zeros((w.B, w.L, w.d), dtype=torch.float32, device="cuda")
    ws = torch.empty(C.crc_fused_workspace_bytes(p), dtype=torch.uint8, device="cuda")
    st = C.State(p)
    idx = list(streams)
    g_set, g_mis, g_pro = [], [], []
    try:
        for c in range(TC // CH):
            t0 = c * CH
            att = np.zeros((w.B, CH, w.L), np.uint8)
            att[idx] = cert["attempts"][:, t0:t0 + CH]
            C.synth_hidden(w.B, CH, w.L, w.d, seed=0, rho_t=w.rho_t, rho_l=w.rho_l, t0=t0,
                           carry=carry, attempts=torch.from_numpy(att).cuda(), out=hbuf)
            for i, b in enumerate(idx):
                ref = torch.from_numpy(cert["hidden"][i, t0:t0 + CH].view(np.int16)).cuda()
                assert torch.equal(hbuf[b].view(torch.int16), ref), (b, c)
            tr = C.Trace.alloc(p, CH, rank_order=False, topk_set=True)
            C.crc_profile_begin()
            C.route_and_cache(p, hbuf, Wd, st, tr, workspace=ws)
            assert C.crc_profile_end()["fused"]["launches"] == 1
            g_set.append(tr.topk_set[idx].cpu().numpy().view(np.uint32))
            g_mis.append(tr.misses[idx].cpu().numpy())
            g_pro.append(tr.proactive[idx].cpu().numpy())
            del tr
    finally:
        del hbuf, ws, carry
        torch.cuda.empty_cache()
    r = st.read(want_caches=True, want_retention=True, want_chain_counters=True)
    assert r["error"] == 0 and r["tokens"] == TC
    g_set, g_mis, g_pro = (np.concatenate(x, axis=1) for x in (g_set, g_mis, g_pro))
    o_set = _sets(cert["topk"], w.N)
    for i, b in enumerate(idx):
        for l in range(w.L):
            bad = np.flatnonzero(~cert["certified"][i, :, l])
            stop = int(bad[0]) if len(bad) else TC
            sl = slice(0, stop)
            assert np.array_equal(g_set[i, sl, l], o_set[i, sl, l]), (b, l)
            assert np.array_equal(g_mis[i, sl, l], cert["misses"][i, sl, l]), (b, l)
            assert np.array_equal(g_pro[i, sl, l], cert["proactive"][i, sl, l]), (b, l)
            if stop == TC:
                assert np.array_equal(r["cache_bits"][b, l], cert["cache_bits"][i, l])
                assert np.array_equal(r["chain_counters"][b, l], cert["counters"][i, l])
                ref = cert["aT"][i, l]
                assert (np.abs(r["retention"][b, l].astype(np.float64) - ref) / ref).max() <= TOL
