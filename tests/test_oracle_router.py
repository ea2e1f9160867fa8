"""Pins of the oracle's router heads: p^X = softmax(W^X_l h) (Sec. 2, 3.2, 3.3)."""
import numpy as np
import pytest
import scipy.special

import crc_synth as S


def _f(bits):
    return S.bf16_bits_to_f32(bits).astype(np.float64)


def test_rows_are_distributions(oracle_lib):
    w = S.TINY.with_(T=16)
    p = oracle_lib.router_probs(S.hidden(w), S.weights(w), w.N)
    assert p.shape == (w.B, w.T, w.L, 3, w.N)
    assert np.all(p > 0)
    assert np.max(np.abs(p.sum(-1) - 1.0)) < 1e-12


def test_matches_library_softmax_of_library_matmul(oracle_lib):
    # Special case reducing to library routines: numpy's matmul in fp64 on the
    # exactly-widened bf16 values, then scipy's softmax.  Distinct heads,
    # layers, tokens and streams catch a transposed operand or a wrong stride.
    w = S.TINY.with_(B=3, T=5, L=3, N=16, d=96)
    h, W = S.hidden(w, seed=1), S.weights(w, seed=2)
    p = oracle_lib.router_probs(h, W, w.N)
    hf, Wf = _f(h), _f(W)
    for b in range(w.B):
        for t in range(w.T):
            for l in range(w.L):
                z = Wf[l] @ hf[b, t, l]                      # [3N]
                ref = scipy.special.softmax(z.reshape(3, w.N), axis=-1)
                assert np.allclose(p[b, t, l], ref, rtol=1e-12, atol=0)


def test_zero_weights_give_uniform(oracle_lib):
    w = S.TINY.with_(B=1, T=2, L=2)
    W = np.zeros((w.L, 3 * w.N, w.d), np.uint16)
    p = oracle_lib.router_probs(S.hidden(w), W, w.N)
    assert np.all(p == 1.0 / w.N)


def test_large_logits_do_not_overflow(oracle_lib):
    # logits around +-3000: a softmax without the max shift would overflow exp.
    N, d = 16, 64
    h = np.zeros(d, np.float32)
    h[0] = 64.0
    W = np.zeros((3 * N, d), np.float32)
    W[:, 0] = np.linspace(-48, 48, 3 * N).astype(np.float32)
    p = oracle_lib.unit_probs(S.bf16_rne_bits(h), S.bf16_rne_bits(W), N)
    z = (S.bf16_bits_to_f32(S.bf16_rne_bits(W)).astype(np.float64) @
         S.bf16_bits_to_f32(S.bf16_rne_bits(h)).astype(np.float64)).reshape(3, N)
    assert np.all(np.isfinite(p))
    assert np.allclose(p, scipy.special.softmax(z, axis=-1), rtol=1e-12, atol=1e-300)


def test_two_expert_logistic_closed_form(oracle_lib):
    # N = 2: p_0 = 1 / (1 + exp(z_1 - z_0)) -- checked through tanh.
    d = 8
    h = S.bf16_rne_bits(np.array([1, 0.5, -2, 0, 0, 0, 0, 0.25], np.float32))
    W = S.bf16_rne_bits(np.array([[0.5, 1, 0, 0, 0, 0, 0, 1]] * 3 +
                                 [[-0.25, 0, 0.75, 0, 0, 0, 0, 0]] * 3, np.float32)[[0, 3, 1, 4, 2, 5]])
    p = oracle_lib.unit_probs(h, W, 2)
    hf, Wf = _f(h), _f(W)
    for head in range(3):
        dz = Wf[2 * head] @ hf - Wf[2 * head + 1] @ hf
        assert abs(p[head, 0] - 0.5 * (1 + np.tanh(dz / 2))) < 1e-15


def test_heads_order_and_copy_init(oracle_lib):
    # Copy initialisation (Sec. 3.4): W^T_l = W^R_l gives p^T == p^R exactly;
    # with identical hidden states across layers (rho_l = 1) and
    # W^S_l = W^R_{l+1}, the Spatio head at layer l-1 equals p^R at layer l.
    w = S.TINY.with_(T=6, rho_l=1.0)
    h = S.hidden(w)
    W = S.weights(w, copy_init=True)
    p = oracle_lib.router_probs(h, W, w.N)
    assert np.array_equal(p[:, :, :, 1], p[:, :, :, 0])
    for l in range(1, w.L):
        assert np.array_equal(p[:, :, l - 1, 2], p[:, :, l, 0])
    assert np.array_equal(p[:, :, w.L - 1, 2], p[:, :, 0, 0])   # wrap-around W^S_L = W^R_1


def test_two_head_mode_leaves_spatio_untouched(oracle_lib):
    w = S.TINY.with_(T=4)
    p2 = oracle_lib.router_probs(S.hidden(w), S.weights(w), w.N, H=2)
    p3 = oracle_lib.router_probs(S.hidden(w), S.weights(w), w.N, H=3)
    assert np.all(p2[:, :, :, 2] == 0)
    assert np.array_equal(p2[:, :, :, :2], p3[:, :, :, :2])
