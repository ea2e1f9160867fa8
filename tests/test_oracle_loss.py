"""The oracle's soft Top-B cache-coverage losses (Sec. 3.1-3.3), pinned to:

* central finite differences of w_T L_T + w_ST L_ST with respect to every
  logit of every head, p^R moving both as a priority term and as a target
  (the gradient is computed analytically by the oracle);
* the tau -> 0 limit, where m_e becomes the hard Top-B indicator (1/2 at the
  B-th element itself), so l = target mass outside the top B + half the
  target mass of the B-th element, computed here from a plain sort;
* validity: l^T vanishes at the last token and l^ST at the first, 0 <= l <= 1,
  and each head's logit gradient sums to zero (softmax is shift-invariant).
"""
import numpy as np
import pytest


def softmax(z):
    e = np.exp(z - z.max(-1, keepdims=True))
    return e / e.sum(-1, keepdims=True)


def test_gradient_matches_finite_differences(oracle_lib):
    rng = np.random.default_rng(1)
    B, T, L, N, Btop, tau = 1, 4, 2, 8, 3, 0.5
    z = rng.normal(size=(B, T, L, 3, N))
    wT, wST = 0.7, 1.3

    def objective(zz):
        r = oracle_lib.cache_loss(softmax(zz).astype(np.float32), Btop, tau, wT, wST, grad=False)
        return wT * r["L_T"] + wST * r["L_ST"]

    g = oracle_lib.cache_loss(softmax(z).astype(np.float32), Btop, tau, wT, wST)["grad"]
    h = 1e-2
    checked = 0
    for idx in np.ndindex(z.shape):
        zp, zm = z.copy(), z.copy()
        zp[idx] += h
        zm[idx] -= h
        fd = (objective(zp) - objective(zm)) / (2 * h)
        assert fd == pytest.approx(g[idx], rel=2e-2, abs=2e-5), idx
        checked += 1
    assert checked == z.size


def test_hard_limit(oracle_lib):
    rng = np.random.default_rng(2)
    B, T, L, N, Btop = 2, 5, 3, 16, 5
    p = softmax(rng.normal(size=(B, T, L, 3, N))).astype(np.float32)
    r = oracle_lib.cache_loss(p, Btop, 1e-7, grad=False)
    for b in range(B):
        for t in range(T):
            for l in range(L):
                if t + 1 < T:
                    s = (p[b, t, l, 0] + p[b, t, l, 1]).astype(np.float32)
                    q = p[b, t + 1, l, 0].astype(np.float64)
                    order = sorted(range(N), key=lambda e: (-float(s[e]), e))
                    want = q[order[Btop:]].sum() + 0.5 * q[order[Btop - 1]]
                    assert r["loss"][b, t, l, 0] == pytest.approx(want, abs=1e-6)
                if t >= 1:
                    a = (p[b, t - 1, l, 0] + p[b, t - 1, l, 1]).astype(np.float32)
                    src = p[b, t, l - 1, 2] if l > 0 else p[b, t - 1, L - 1, 2]
                    s = (a + src).astype(np.float32)
                    q = p[b, t, l, 0].astype(np.float64)
                    order = sorted(range(N), key=lambda e: (-float(s[e]), e))
                    want = q[order[Btop:]].sum() + 0.5 * q[order[Btop - 1]]
                    assert r["loss"][b, t, l, 1] == pytest.approx(want, abs=1e-6)


def test_validity_range_and_shift_invariance(oracle_lib):
    rng = np.random.default_rng(3)
    p = softmax(rng.normal(size=(3, 7, 4, 3, 32))).astype(np.float32)
    r = oracle_lib.cache_loss(p, 8, 0.05)
    assert np.all(r["loss"][:, -1, :, 0] == 0) and np.all(r["loss"][:, 0, :, 1] == 0)
    assert np.all(r["loss"] >= 0) and np.all(r["loss"] <= 1)
    # up to the fp32 probabilities' rounding (they sum to 1 within ~1e-7)
    assert np.abs(r["grad"].sum(-1)).max() < 1e-9
    # the means are over the valid positions only
    n = 3 * 6 * 4
    assert r["L_T"] == pytest.approx(r["loss"][..., 0].astype(np.float64).sum() / n, rel=1e-12)
