"""GPU parity of the soft Top-B coverage losses (crc_cache_loss) against the
oracle (oracle.cache_loss) on the same fp32 probabilities.

Tolerances, from the arithmetic: both sides form the priorities by the same
fp32 additions, so theta_B and the element carrying its subgradient are the
same decision; the kernel's sigmoid (hardware exponential, fast divide) and
its sums are fp32, the oracle's fp64.  A per-position loss is a q-weighted
sum of terms in [0, 1], so it is compared to 2e-5 absolute.  A gradient
element dz_e = p_e (d_e - <p, d>) carries fp32 error from d (a few terms of
relative error ~1e-6 each, and the theta term, a sum of N of them) and from
<p, d> (N products), so it is compared to 1e-4 of its row's largest entry
plus 3e-5 p_e max|d| of the row (d from the oracle).  A dropped or misplaced
term moves entries by O(1) of their size.
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


def problem(C, B, L, N):
    return C.problem(L=L, N=N, K=1, d=16, C=1, R=0, B=B, expert_bytes=1)


def run(C, p32, top_b, tau, w_T=1.0, w_ST=1.0, heads=3, grad=True):
    B, T, L, _, N = p32.shape
    pr = problem(C, B, L, N)
    probs = torch.from_numpy(p32).cuda()
    loss, means, g = C.cache_loss(pr, probs, top_b, tau, w_T, w_ST, heads=heads, grad=grad)
    torch.cuda.synchronize()
    assert C.crc_device_error() == 0
    return (loss.cpu().numpy(), means.cpu().numpy(),
            None if g is None else g.cpu().numpy())


def check_grad(got, o, p32, heads=3):
    want, dp = o["grad"], o["grad_p"]
    hs = slice(0, heads)
    w, d, p, g = want[..., hs, :], dp[..., hs, :], p32[..., hs, :].astype(np.float64), got[..., hs, :]
    tol = 1e-4 * np.abs(w).max(-1, keepdims=True) + 3e-5 * p * np.abs(d).max(-1, keepdims=True)
    bad = np.abs(g - w) > tol + 1e-30
    assert not bad.any(), (np.argwhere(bad)[:5], g[bad][:5], w[bad][:5])


def check(C, oracle_lib, p32, top_b, tau, w_T=1.0, w_ST=1.0, heads=3):
    loss, means, g = run(C, p32, top_b, tau, w_T, w_ST, heads)
    o = oracle_lib.cache_loss(p32, top_b, tau, w_T, w_ST if heads == 3 else 0.0, grad_p=True)
    np.testing.assert_allclose(loss[..., 0], o["loss"][..., 0], rtol=0, atol=2e-5)
    if heads == 3:
        np.testing.assert_allclose(loss[..., 1], o["loss"][..., 1], rtol=0, atol=2e-5)
        assert means[1] == pytest.approx(o["L_ST"], rel=1e-5, abs=1e-7)
    else:
        assert np.all(loss[..., 1] == 0) and means[1] == 0
    assert means[0] == pytest.approx(o["L_T"], rel=1e-5, abs=1e-7)
    check_grad(g, o, p32, heads)
    return loss, means, g


CASES = [  # name, B, T, L, N, top_b, tau, quant
    ("qwen3", 2, 40, 3, 128, 20, 0.03, None),
    ("gptoss", 3, 50, 4, 32, 8, 0.05, None),
    ("tiny", 2, 64, 4, 16, 3, 0.05, None),
    ("n48", 2, 33, 2, 48, 5, 0.1, None),
    ("n96", 1, 37, 3, 96, 11, 0.03, None),
    ("n256", 1, 20, 2, 256, 40, 0.02, None),
    ("ties", 2, 40, 3, 64, 8, 0.05, 32),
    ("ties_n128", 2, 30, 2, 128, 20, 0.03, 64),
    ("b1", 2, 30, 2, 128, 1, 0.03, None),
    ("bN", 1, 30, 2, 32, 32, 0.05, None),
    # short rows (N = 16, 32 with top_b <= 16): one or two lanes per row
    ("n32_ties", 2, 40, 3, 32, 8, 0.05, 16),
    ("n32_ties_fine", 2, 40, 3, 32, 6, 0.05, 256),
    ("n32_b16", 2, 40, 3, 32, 16, 0.05, None),
    ("n32_b1", 2, 30, 2, 32, 1, 0.05, None),
    ("n32_b3", 3, 33, 5, 32, 3, 0.1, None),
    ("n32_b17", 1, 30, 2, 32, 17, 0.05, None),
    ("n16_ties", 2, 40, 3, 16, 5, 0.05, 8),
    ("n16_b16", 2, 30, 2, 16, 16, 0.05, None),
]


@pytest.mark.parametrize("name,B,T,L,N,top_b,tau,quant", CASES, ids=[c[0] for c in CASES])
def test_loss_and_gradient_match_oracle(C, oracle_lib, name, B, T, L, N, top_b, tau, quant):
    p32 = S.distributions(B, T, L, N, seed=sum(map(ord, name)), quant=quant)
    check(C, oracle_lib, p32, top_b, tau, w_T=0.7, w_ST=1.3)


@pytest.mark.parametrize("N,top_b", [(128, 20), (32, 8)])
@pytest.mark.parametrize("kind", ["uncorrelated", "repeated", "repeated_ties"])
def test_theta_guess_extremes(C, oracle_lib, kind, N, top_b):
    """theta_B starts from the previous token's: far off when consecutive
    tokens are unrelated, exact when they repeat (with ties at theta too).
    N = 32 runs the short-row kernel on the same extremes."""
    if kind == "uncorrelated":
        p32 = S.distributions(2, 60, 3, N, seed=13, rho=0.0)
    else:
        p32 = np.repeat(S.distributions(2, 1, 3, N, seed=14,
                                        quant=N // 2 if kind == "repeated_ties" else None), 50,
                        axis=1)
    check(C, oracle_lib, np.ascontiguousarray(p32), top_b, 0.03)


@pytest.mark.parametrize("w_T,w_ST", [(0.0, 1.0), (1.0, 0.0), (0.1, 0.0)])
def test_objective_weights(C, oracle_lib, w_T, w_ST):
    """The paper's full mode trains L_ST alone, the update-only mode L_T alone."""
    p32 = S.distributions(2, 45, 3, 128, seed=7)
    check(C, oracle_lib, p32, 20, 0.03, w_T, w_ST)


@pytest.mark.parametrize("N,top_b", [(128, 20), (32, 8)])
def test_update_only_heads_2(C, oracle_lib, N, top_b):
    """heads = 2 never reads the S head (NaN here) and leaves its gradient rows."""
    p32 = S.distributions(2, 45, 3, N, seed=8)
    check(C, oracle_lib, p32, top_b, 0.03, heads=2)
    nan_s = p32.copy()
    nan_s[..., 2, :] = np.nan
    pr = problem(C, 2, 3, N)
    probs = torch.from_numpy(nan_s).cuda()
    grad = torch.full(probs.shape, 7.0, device="cuda")
    loss, means, _ = C.cache_loss(pr, probs, top_b, 0.03, heads=2, grad_out=grad)
    g = grad.cpu().numpy()
    assert np.all(g[..., 2, :] == 7.0)
    ref = run(C, p32, top_b, 0.03, heads=2)
    assert np.array_equal(loss.cpu().numpy(), ref[0])
    assert np.array_equal(g[..., :2, :], ref[2][..., :2, :])


@pytest.mark.parametrize("T", [1, 2, 3, 17])
def test_short_sequences(C, oracle_lib, T):
    p32 = S.distributions(3, T, 2, 32, seed=T)
    loss, means, g = check(C, oracle_lib, p32, 4, 0.05)
    if T == 1:
        assert np.all(loss == 0) and np.all(means == 0) and np.all(g == 0)


@pytest.mark.parametrize("N,top_b", [(128, 20), (32, 8)])
def test_chunks_and_halos(C, oracle_lib, N, top_b):
    """One stream over two layers splits its tokens into chunks, each with a
    halo step.  T = 300 makes 10 chunks of 30 tokens; the first 250 tokens
    alone make 8 chunks of 32, and give the same values wherever the two
    sequences see the same neighbours (the coefficients matched).  At N = 32
    the two chains of a chunk share a warp with 14 idle row pairs."""
    p32 = S.distributions(1, 300, 2, N, seed=9)
    la, _, ga = check(C, oracle_lib, p32, top_b, 0.03)
    w = 249 / 299                                          # same w / (B (T - 1) L)
    lb, _, gb = run(C, np.ascontiguousarray(p32[:, :250]), top_b, 0.03, w_T=w, w_ST=w)
    assert np.array_equal(la[:, :249, :, 0], lb[:, :249, :, 0])
    assert np.array_equal(la[:, :250, :, 1], lb[:, :250, :, 1])
    np.testing.assert_allclose(gb[:, :249], ga[:, :249], rtol=1e-6, atol=1e-12)


@pytest.mark.parametrize("N,top_b", [(128, 20), (32, 8)])
def test_forward_only_and_determinism(C, N, top_b):
    p32 = S.distributions(4, 80, 6, N, seed=10)
    l1, m1, g1 = run(C, p32, top_b, 0.03)
    l2, m2, g2 = run(C, p32, top_b, 0.03)
    l3, m3, _ = run(C, p32, top_b, 0.03, grad=False)
    assert np.array_equal(l1, l2) and np.array_equal(m1, m2) and np.array_equal(g1, g2)
    assert np.array_equal(l1, l3) and np.array_equal(m1, m3)


def test_argument_errors(C):
    pr = problem(C, 1, 2, 32)
    probs = torch.zeros((1, 4, 2, 3, 32), device="cuda")
    for kw in ({"top_b": 0}, {"top_b": 33}, {"tau": 0.0}, {"tau": float("nan")},
               {"w_T": float("inf")}, {"heads": 1}):
        args = dict(top_b=4, tau=0.05, w_T=1.0, w_ST=1.0, heads=3)
        args.update(kw)
        with pytest.raises(C.CrcError):
            C.cache_loss(pr, probs, **args)


def sampled_windows(T, n, rng):
    starts = sorted(set([0, T - 12] + list(rng.integers(1, T - 12, size=n))))
    return [(a, min(T, a + 12)) for a in starts]


@pytest.mark.parametrize("w", [S.QWEN3_30B, S.GPT_OSS_20B], ids=["qwen3", "gptoss"])
def test_full_size_sampled(C, oracle_lib, w):
    """The paper's settings, (B, tau) = (20, 0.03) for Qwen3 and (8, 0.05) for
    GPT-OSS, at the full stream x token x layer size in the launch the bench
    times; sampled token windows of sampled streams against the oracle, and
    properties of the whole output."""
    top_b, tau = (20, 0.03) if w.N == 128 else (8, 0.05)
    B, T, L, N = w.B, w.T, w.L, w.N
    pr = problem(C, B, L, N)
    probs = torch.empty((B, T, L, 3, N), dtype=torch.float32, device="cuda")
    for b0 in range(0, B, 8):
        probs[b0:b0 + 8] = torch.from_numpy(
            S.distributions(B, T, L, N, seed=11, streams=range(b0, min(B, b0 + 8)))).cuda()
    loss, means, grad = C.cache_loss(pr, probs, top_b, tau, 1.0, 1.0)
    torch.cuda.synchronize()
    n_full = B * (T - 1) * L
    lt = loss.double()
    assert means[0].item() == pytest.approx(lt[..., 0].sum().item() / n_full, rel=1e-9)
    assert means[1].item() == pytest.approx(lt[..., 1].sum().item() / n_full, rel=1e-9)
    rowsum = grad.sum(-1).abs().max().item()
    assert rowsum <= 1e-4 * grad.abs().max().item()          # softmax shift invariance
    rng = np.random.default_rng(12)
    for b in sorted(set([0, B - 1] + list(rng.integers(1, B - 1, size=2)))):
        pb = S.distributions(B, T, L, N, seed=11, streams=[b])
        for ta, tb in sampled_windows(T, 3, rng):
            lo, hi = max(0, ta - 1), min(T, tb + 1)
            sub = pb[:, lo:hi]
            n_sub = (hi - lo - 1) * L
            o = oracle_lib.cache_loss(sub, top_b, tau, n_sub / n_full, n_sub / n_full,
                                      grad_p=True)
            k0, k1 = ta - lo, tb - lo
            got_l = loss[b, ta:tb].cpu().numpy()
            np.testing.assert_allclose(got_l, o["loss"][0, k0:k1], rtol=0, atol=2e-5)
            got_g = grad[b:b + 1, ta:tb].cpu().numpy()
            check_grad(got_g, {"grad": o["grad"][:, k0:k1], "grad_p": o["grad_p"][:, k0:k1]},
                       sub[:, k0:k1])
