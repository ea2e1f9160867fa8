"""GPU parity: the CUDA path through the C ABI against the CPU oracle.

* router heads vs the fp64 oracle: relative error <= 1e-3 (the stated fp32
  tolerance), plus a cuBLAS cross-check;
* cache scan vs the oracle's literal fp32 scan fed the SAME fp32
  probabilities (the oracle's own fp64 probabilities rounded to fp32):
  bit-exact Top-K trace, misses, proactive loads, caches, carried scores,
  counters -- ties included, since both sides use one total order;
* chunked calls == one call; route_and_cache == route_scores + cache_scan;
* end to end vs the fp64 oracle up to each chain's first near-tie decision
  (relative decision margin < 1e-3, flagged by the oracle);
* the device input generator reproduces the host generator bit for bit;
* the full Qwen3-30B-shaped workload in the benchmark's launch
  configuration: sampled router rows vs the oracle, one whole stream's scan
  vs the oracle, invariants on every chain.
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


def dev_bf16(bits: np.ndarray):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).cuda()


def host_bits(t) -> np.ndarray:
    return t.view(torch.int16).cpu().numpy().view(np.uint16)


def rel_err(gpu, ref):
    return np.abs(gpu.astype(np.float64) - ref) / np.maximum(np.abs(ref), 1e-30)


def gpu_scan(C, w, probs32, chunks=None):
    p = C.problem_of(w)
    st = C.State(p)
    T = probs32.shape[1]
    tr = C.Trace.alloc(p, T)
    sc = torch.from_numpy(np.ascontiguousarray(probs32)).cuda()
    if chunks is None:
        C.cache_scan(p, sc, st, tr)
    else:
        t0 = 0
        for n in chunks:
            sub = sc[:, t0:t0 + n].contiguous()
            part = C.Trace.alloc(p, n)
            C.cache_scan(p, sub, st, part)
            tr.topk[:, t0:t0 + n] = part.topk
            tr.misses[:, t0:t0 + n] = part.misses
            tr.proactive[:, t0:t0 + n] = part.proactive
            t0 += n
    r = st.read(want_caches=True, want_retention=True, want_chain_counters=True)
    r.update(topk=tr.topk.cpu().numpy(), misses=tr.misses.cpu().numpy(),
             proactive=tr.proactive.cpu().numpy())
    return r


def assert_scan_equal(g, o, tag=""):
    assert np.array_equal(g["topk"], o["topk"]), tag + " topk"
    assert np.array_equal(g["misses"], o["misses"]), tag + " misses"
    assert np.array_equal(g["proactive"], o["proactive"]), tag + " proactive"
    assert np.array_equal(g["cache_bits"], o["cache_bits"]), tag + " caches"
    assert np.array_equal(g["retention"].view(np.uint32), o["aT"].view(np.uint32)), tag + " s^T"
    assert np.array_equal(g["chain_counters"], o["counters"]), tag + " counters"


# --------------------------------------------------------------------------- #
ROUTER_CASES = [
    S.TINY,                                                          # N=16
    S.TINY.with_(N=32, K=4, C=8, R=2, d=200, B=3, T=37, L=3),        # partial K block, ragged T
    S.TINY.with_(N=64, K=4, C=16, R=3, d=512, B=2, T=70, L=2),
    S.QWEN3_30B.with_(B=2, T=130, L=3),                              # N=128, two token tiles
    S.GPT_OSS_20B.with_(B=5, T=9, L=2),                              # d=2880, small T: multi-stream tiles
]


@pytest.mark.parametrize("w", ROUTER_CASES, ids=lambda w: f"N{w.N}-d{w.d}-B{w.B}-T{w.T}")
@pytest.mark.parametrize("heads", [3, 2])
def test_route_scores_vs_oracle(C, oracle_lib, w, heads):
    h, W = S.hidden(w, seed=1), S.weights(w, seed=2)
    ref = oracle_lib.router_probs(h, W, w.N, H=heads)
    p = C.problem_of(w)
    out = torch.full((w.B, w.T, w.L, 3, w.N), -7.0, device="cuda")
    C.route_scores(p, dev_bf16(h), dev_bf16(W), heads=heads, out=out)
    assert C.crc_device_error() == 0
    g = out.cpu().numpy()
    err = rel_err(g[:, :, :, :heads], ref[:, :, :, :heads])
    assert err.max() <= TOL, err.max()
    assert err.max() <= 2.5e-4                      # leaves room under the 1e-3 margin filter
    if heads == 2:
        assert np.all(g[:, :, :, 2] == -7.0)        # S slot untouched
    # library cross-check: cuBLAS fp32 GEMM on the widened bf16 values + torch softmax
    hf = dev_bf16(h).float()
    Wf = dev_bf16(W).float()
    z = torch.einsum("btld,lkd->btlk", hf, Wf).view(w.B, w.T, w.L, 3, w.N)
    sm = torch.softmax(z, dim=-1).cpu().numpy()
    assert rel_err(g[:, :, :, :heads], sm[:, :, :, :heads]).max() <= TOL


# --------------------------------------------------------------------------- #
def _oracle_probs32(oracle_lib, w, seed=0, quant=None):
    h, W = S.hidden(w, seed=seed), S.weights(w, seed=seed + 100)
    p = oracle_lib.router_probs(h, W, w.N, H=3 if w.R > 0 else 2)
    if quant:                       # coarse values: many exact ties
        p = np.round(p * quant) / quant
    return p.astype(np.float32)


SCAN_CASES = [
    ("tiny", S.TINY, None),
    ("tiny-r0", S.TINY.with_(R=0), None),
    ("qwen3", S.QWEN3_30B.with_(B=3, T=96, L=4), None),
    ("gptoss", S.GPT_OSS_20B.with_(B=4, T=128, L=3, d=512), None),
    ("c96-r0", S.QWEN3_30B.with_(B=2, T=64, L=3, C=96, R=0), None),
    ("r16", S.QWEN3_30B.with_(B=2, T=64, L=2, R=16), None),
    ("c-eq-k", S.GPT_OSS_20B.with_(B=3, T=64, L=2, d=256, C=4, K=4), None),
    ("c-eq-n", S.TINY.with_(C=16, R=3), None),
    ("k1", S.TINY.with_(K=1, C=1, R=2), None),
    ("ties-n16", S.TINY.with_(R=2), 16),
    ("ties-n128", S.QWEN3_30B.with_(B=2, T=48, L=3, d=256), 64),
]


@pytest.mark.parametrize("name,w,quant", SCAN_CASES, ids=[c[0] for c in SCAN_CASES])
def test_cache_scan_untraced_state_bit_exact(C, oracle_lib, name, w, quant):
    # Without a trace the scan takes the Top-K set from its batched selection
    # instead of rank-ordered pops; the caches and counters must not change.
    p32 = _oracle_probs32(oracle_lib, w, quant=quant)
    p = C.problem_of(w)
    st = C.State(p)
    C.cache_scan(p, torch.from_numpy(p32).cuda(), st, None)
    g = st.read(want_caches=True, want_retention=True, want_chain_counters=True)
    o = oracle_lib.scan(p32, w.K, w.C, w.R, trace=False)
    assert np.array_equal(g["cache_bits"], o["cache_bits"])
    assert np.array_equal(g["chain_counters"], o["counters"])
    assert np.array_equal(g["retention"].view(np.uint32), o["aT"].view(np.uint32))


@pytest.mark.parametrize("name,w,quant", SCAN_CASES, ids=[c[0] for c in SCAN_CASES])
def test_cache_scan_bit_exact(C, oracle_lib, name, w, quant):
    p32 = _oracle_probs32(oracle_lib, w, quant=quant)
    g = gpu_scan(C, w, p32)
    o = oracle_lib.scan(p32, w.K, w.C, w.R)
    assert_scan_equal(g, o, name)
    c = g["chain_counters"]
    assert np.all(c[..., 0] + c[..., 1] == w.T * w.K)
    assert g["error"] == 0 and g["tokens"] == w.T


@pytest.mark.parametrize("N,K,C_,R", [(256, 8, 32, 4), (96, 6, 20, 15), (48, 2, 5, 3),
                                      (64, 13, 20, 2), (128, 32, 40, 3), (32, 1, 1, 1)])
def test_cache_scan_wide_and_odd_n(C, oracle_lib, N, K, C_, R):
    # scan-only sizes the router does not take; probability-like synthetic scores
    w = S.TINY.with_(N=N, K=K, C=C_, R=R, B=3, T=80, L=3)
    p32 = S.near_uniform_scores((w.B, w.T, w.L, 3, N), seed=N)
    g = gpu_scan(C, w, p32)
    o = oracle_lib.scan(p32, K, C_, R)
    assert_scan_equal(g, o, f"N{N}")
    p = C.problem_of(w)
    st = C.State(p)
    C.cache_scan(p, torch.from_numpy(p32).cuda(), st, None)
    u = st.read(want_caches=True, want_chain_counters=True)
    assert np.array_equal(u["cache_bits"], o["cache_bits"])
    assert np.array_equal(u["chain_counters"], o["counters"])


def test_chunked_calls_equal_one_call(C, oracle_lib):
    w = S.QWEN3_30B.with_(B=2, T=100, L=3, d=256)
    p32 = _oracle_probs32(oracle_lib, w, seed=3)
    one = gpu_scan(C, w, p32)
    parts = gpu_scan(C, w, p32, chunks=[1, 16, 50, 33])
    for k in ("topk", "misses", "proactive", "cache_bits", "chain_counters"):
        assert np.array_equal(one[k], parts[k]), k
    assert np.array_equal(one["retention"], parts["retention"])
    assert parts["tokens"] == w.T
    assert_scan_equal(parts, oracle_lib.scan(p32, w.K, w.C, w.R), "chunked")


@pytest.mark.parametrize("w", [S.TINY, S.QWEN3_30B.with_(B=2, T=70, L=3),
                               S.GPT_OSS_20B.with_(B=3, T=40, L=2, d=576),
                               S.QWEN3_30B.with_(B=2, T=33, L=2, R=0)],
                         ids=["tiny", "qwen3", "gptoss", "r0"])
def test_route_and_cache_equals_pair(C, w):
    p = C.problem_of(w)
    h = dev_bf16(S.hidden(w, seed=5))
    W = dev_bf16(S.weights(w, seed=6))
    heads = 3 if w.R > 0 else 2
    scores = C.route_scores(p, h, W, heads=heads)
    st_pair = C.State(p)
    tr_pair = C.Trace.alloc(p, w.T)
    C.cache_scan(p, scores, st_pair, tr_pair)
    ref = st_pair.read(want_caches=True, want_retention=True, want_chain_counters=True)
    for chunk in (1, 7, w.T):
        st = C.State(p)
        tr = C.Trace.alloc(p, w.T)
        ws = torch.empty(C.crc_workspace_bytes(p, chunk), dtype=torch.uint8, device="cuda")
        C.route_and_cache(p, h, W, st, tr, workspace=ws)
        got = st.read(want_caches=True, want_retention=True, want_chain_counters=True)
        for k in ("cache_bits", "chain_counters", "retention"):
            assert np.array_equal(got[k], ref[k]), (chunk, k)
        assert torch.equal(tr.topk, tr_pair.topk) and torch.equal(tr.misses, tr_pair.misses)
        assert torch.equal(tr.proactive, tr_pair.proactive)
        assert got["tokens"] == w.T and got["error"] == 0


def test_end_to_end_vs_fp64_oracle_on_certified_prefixes(C, oracle_lib):
    w = S.TINY
    h, W = S.hidden(w, seed=11), S.weights(w, seed=12)
    o = oracle_lib.run(h, W, w.N, w.K, w.C, w.R)
    p = C.problem_of(w)
    st = C.State(p)
    tr = C.Trace.alloc(p, w.T)
    C.route_and_cache(p, dev_bf16(h), dev_bf16(W), st, tr)
    topk, mis, pro = tr.topk.cpu().numpy(), tr.misses.cpu().numpy(), tr.proactive.cpu().numpy()
    covered = 0
    for b in range(w.B):
        for l in range(w.L):
            # chains interact only through router scores, never through
            # decisions: a near-tie ends the certified prefix of its own chain
            flags = o["margins"][b, :, l] < TOL
            stop = int(np.argmax(flags)) if flags.any() else w.T
            covered += stop
            sl = slice(0, stop)
            assert np.array_equal(np.sort(topk[b, sl, l], -1), np.sort(o["topk"][b, sl, l], -1))
            assert np.array_equal(mis[b, sl, l], o["misses"][b, sl, l])
            assert np.array_equal(pro[b, sl, l], o["proactive"][b, sl, l])
    assert covered >= 0.2 * w.B * w.T * w.L


# --------------------------------------------------------------------------- #
@pytest.mark.parametrize("w", [S.TINY, S.GPT_OSS_20B.with_(B=3, T=20, L=5, d=2880)],
                         ids=["tiny", "gptoss"])
def test_device_generator_matches_host_generator(C, w):
    Wd = C.synth_weights(w.L, w.N, w.d, seed=7)
    assert np.array_equal(host_bits(Wd), S.weights(w, seed=7))
    Wc = C.synth_weights(w.L, w.N, w.d, seed=7, copy_init=True)
    assert np.array_equal(host_bits(Wc), S.weights(w, seed=7, copy_init=True))
    ref = S.hidden(w, seed=9)
    hd, _ = C.synth_hidden(w.B, w.T, w.L, w.d, seed=9, rho_t=w.rho_t, rho_l=w.rho_l)
    assert np.array_equal(host_bits(hd), ref)
    # chunked generation carries the token recurrence
    carry = None
    parts = []
    for t0, n in ((0, 3), (3, w.T - 3)):
        hp, carry = C.synth_hidden(w.B, n, w.L, w.d, seed=9, rho_t=w.rho_t, rho_l=w.rho_l,
                                   t0=t0, carry=carry)
        parts.append(host_bits(hp))
    assert np.array_equal(np.concatenate(parts, axis=1), ref)


# --------------------------------------------------------------------------- #
FULL = [S.QWEN3_30B, S.GPT_OSS_20B]


@pytest.mark.parametrize("w", FULL, ids=lambda w: w.name)
def test_full_size_workload(C, oracle_lib, w):
    """The benchmark's workload and launch configuration, checked on samples."""
    p = C.problem_of(w)
    Wd = C.synth_weights(w.L, w.N, w.d, seed=0)
    hd, _ = C.synth_hidden(w.B, w.T, w.L, w.d, seed=0, rho_t=w.rho_t, rho_l=w.rho_l)
    torch.cuda.synchronize()
    W = host_bits(Wd)
    # the fused call exactly as the benchmark issues it
    chunk = 16
    ws = torch.empty(C.crc_workspace_bytes(p, chunk), dtype=torch.uint8, device="cuda")
    st = C.State(p)
    tr = C.Trace.alloc(p, w.T)
    C.route_and_cache(p, hd, Wd, st, tr, workspace=ws)
    fused = st.read(want_caches=True, want_retention=True, want_chain_counters=True)
    assert fused["error"] == 0 and fused["tokens"] == w.T
    cc = fused["chain_counters"]
    assert np.all(cc[..., 0] + cc[..., 1] == w.T * w.K)
    assert int(tr.proactive.max()) <= w.R
    for bits in fused["cache_bits"].reshape(-1, fused["cache_bits"].shape[-1]):
        assert sum(bin(int(x)).count("1") for x in bits) == w.C

    # router rows on sampled units vs the oracle
    heads = 3 if w.R > 0 else 2
    scores = C.route_scores(p, hd, Wd, heads=heads)
    rng = np.random.default_rng(0)
    hb = hd.view(torch.int16)
    for _ in range(48):
        b, t, l = (int(rng.integers(0, w.B)), int(rng.integers(0, w.T)),
                   int(rng.integers(0, w.L)))
        row = hb[b, t, l].cpu().numpy().view(np.uint16)
        ref = oracle_lib.unit_probs(row, W[l], w.N, H=heads)
        assert rel_err(scores[b, t, l, :heads].cpu().numpy(), ref).max() <= TOL

    # the fused kernel (no trace, fused workspace) equals the chunked call on every chain
    wsf = torch.empty(C.crc_fused_workspace_bytes(p), dtype=torch.uint8, device="cuda")
    stf = C.State(p)
    C.crc_profile_begin()
    C.route_and_cache(p, hd, Wd, stf, None, workspace=wsf)
    assert C.crc_profile_end()["fused"]["launches"] == 1
    fz = stf.read(want_caches=True, want_retention=True, want_chain_counters=True)
    assert fz["error"] == 0 and fz["tokens"] == w.T
    assert np.array_equal(fz["cache_bits"], fused["cache_bits"])
    assert np.array_equal(fz["chain_counters"], fused["chain_counters"])
    assert np.array_equal(fz["retention"].view(np.uint32), fused["retention"].view(np.uint32))
    # the same fused kernel writing its per-access trace
    stt = C.State(p)
    trf = C.Trace.alloc(p, w.T, caches=True, rank_order=False, topk_set=True)
    C.crc_profile_begin()
    C.route_and_cache(p, hd, Wd, stt, trf, workspace=wsf)
    assert C.crc_profile_end()["fused"]["launches"] == 1
    ft = stt.read(want_caches=True, want_retention=True, want_chain_counters=True)
    for k in ("cache_bits", "chain_counters"):
        assert np.array_equal(ft[k], fz[k]), k
    assert np.array_equal(ft["retention"].view(np.uint32), fz["retention"].view(np.uint32))
    del wsf

    # fused == pair on every stream, access by access
    st2 = C.State(p)
    tr2 = C.Trace.alloc(p, w.T, caches=True, topk_set=True)
    C.cache_scan(p, scores, st2, tr2)
    pair = st2.read(want_caches=True, want_retention=True, want_chain_counters=True)
    assert np.array_equal(pair["cache_bits"], fused["cache_bits"])
    assert np.array_equal(pair["chain_counters"], fused["chain_counters"])
    assert np.array_equal(pair["retention"].view(np.uint32), fused["retention"].view(np.uint32))
    assert torch.equal(tr.topk, tr2.topk) and torch.equal(tr.misses, tr2.misses)
    for k in ("topk_set", "misses", "proactive", "cache_mid", "cache_after"):
        assert torch.equal(getattr(trf, k), getattr(tr2, k)), k
    del trf

    # one whole stream: host-generated hidden (same bits), oracle probabilities
    # rounded to fp32 in place of that stream's scores, scan vs the oracle
    b = w.B // 2
    hs = S.hidden_stream(0, b, w.T, w.L, w.d, w.rho_t, w.rho_l)
    assert np.array_equal(hs, host_bits(hd[b]))
    p32 = oracle_lib.router_probs(hs[None], W, w.N, H=heads).astype(np.float32)
    scores[b] = torch.from_numpy(p32[0]).cuda()
    st3 = C.State(p)
    tr3 = C.Trace.alloc(p, w.T)
    C.cache_scan(p, scores, st3, tr3)
    g = st3.read(want_caches=True, want_retention=True, want_chain_counters=True)
    o = oracle_lib.scan(p32, w.K, w.C, w.R)
    assert np.array_equal(tr3.topk[b].cpu().numpy(), o["topk"][0])
    assert np.array_equal(tr3.misses[b].cpu().numpy(), o["misses"][0])
    assert np.array_equal(tr3.proactive[b].cpu().numpy(), o["proactive"][0])
    assert np.array_equal(g["cache_bits"][b], o["cache_bits"][0])
    assert np.array_equal(g["retention"][b].view(np.uint32), o["aT"][0].view(np.uint32))
    assert np.array_equal(g["chain_counters"][b], o["counters"][0])


# --------------------------------------------------------------------------- #
FUSED_CASES = [
    ("tiny", S.TINY),                                               # SB=4, TB=32
    ("qwen3", S.QWEN3_30B.with_(T=41, L=5)),                        # SB=32, TB=4, ragged T
    ("gptoss", S.GPT_OSS_20B.with_(B=128, T=23, L=3, d=576)),       # 4 stream groups
    ("r0", S.QWEN3_30B.with_(B=40, T=19, L=4, R=0, C=16)),          # 2 heads, partial group
    ("n64-one-layer", S.TINY.with_(N=64, K=3, C=9, R=5, B=6, T=50, L=1, d=192)),
    ("k1", S.TINY.with_(K=1, C=2, R=2, B=9, T=33)),
    # 128-token tiles of one stream: N = 128 runs on CTA pairs when B is even
    ("pairs-ragged", S.QWEN3_30B.with_(B=4, T=300, L=3, d=256)),     # blocks of 100 | 128, 72
    ("pairs-r0", S.QWEN3_30B.with_(B=6, T=260, L=2, R=0, C=16, d=256)),
    ("pairs-k4", S.QWEN3_30B.with_(B=2, T=256, L=2, K=4, C=12, R=3, d=192)),
    ("odd-b-one-cta", S.QWEN3_30B.with_(B=5, T=200, L=3, d=256)),
]


@pytest.mark.parametrize("name,w", FUSED_CASES, ids=[c[0] for c in FUSED_CASES])
def test_fused_kernel_equals_pair(C, name, w):
    """route_and_cache with a workspace large enough for the fused kernel
    equals route_scores + cache_scan bit for bit, over two calls that continue
    the same streams: without a trace, and with the fused kernel writing its
    per-access trace (Top-K set, misses, proactive loads, the cache after the
    refinement and after UpdateCache), which must equal the pair's element by
    element."""
    p = C.problem_of(w)
    W = dev_bf16(S.weights(w, seed=31))
    h = dev_bf16(S.hidden(w, seed=32))
    heads = 3 if w.R > 0 else 2
    split = [w.T // 3, w.T - w.T // 3]
    st_pair, st_fused, st_traced = C.State(p), C.State(p), C.State(p)
    ws = torch.empty(C.crc_fused_workspace_bytes(p), dtype=torch.uint8, device="cuda")
    tr_pair, tr_fused = [], []
    t0 = 0
    for n in split:
        hc = h[:, t0:t0 + n].contiguous()
        tp = C.Trace.alloc(p, n, caches=True, topk_set=True)
        C.cache_scan(p, C.route_scores(p, hc, W, heads=heads), st_pair, tp)
        C.crc_profile_begin()
        C.route_and_cache(p, hc, W, st_fused, None, workspace=ws)
        kt = C.crc_profile_end()
        assert kt["fused"]["launches"] == 1 and kt["router"]["launches"] == 0
        tf = C.Trace.alloc(p, n, caches=True, rank_order=False, topk_set=True)
        C.crc_profile_begin()
        C.route_and_cache(p, hc, W, st_traced, tf, workspace=ws)
        kt = C.crc_profile_end()
        assert kt["fused"]["launches"] == 1 and kt["router"]["launches"] == 0
        tr_pair.append(tp)
        tr_fused.append(tf)
        t0 += n
    a = st_pair.read(want_caches=True, want_retention=True, want_chain_counters=True)
    for st in (st_fused, st_traced):
        b = st.read(want_caches=True, want_retention=True, want_chain_counters=True)
        assert b["error"] == 0 and b["tokens"] == w.T
        for k in ("cache_bits", "chain_counters"):
            assert np.array_equal(a[k], b[k]), k
        assert np.array_equal(a["retention"].view(np.uint32), b["retention"].view(np.uint32))
    for k in ("topk_set", "misses", "proactive", "cache_mid", "cache_after"):
        g = torch.cat([getattr(x, k) for x in tr_fused], dim=1)
        r = torch.cat([getattr(x, k) for x in tr_pair], dim=1)
        assert torch.equal(g, r), k
