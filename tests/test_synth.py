"""Pins of the seeded input generator (no method arithmetic lives there)."""
import math

import numpy as np
import pytest
import torch

import crc_synth as S


@pytest.mark.parametrize("ctr,key,expect", [
    # Known-answer vectors published with Random123 for philox4x32_10.
    ((0, 0, 0, 0), (0, 0), (0x6627E8D5, 0xE169C58D, 0xBC57AC4C, 0x9B00DBD8)),
    ((0xFFFFFFFF,) * 4, (0xFFFFFFFF,) * 2, (0x408F276D, 0x41C83B0E, 0xA20BC7C6, 0x6D5451FD)),
    ((0x243F6A88, 0x85A308D3, 0x13198A2E, 0x03707344), (0xA4093822, 0x299F31D0),
     (0xD16CFE09, 0x94FDCCEB, 0x5001E420, 0x24126EA1)),
])
def test_philox_known_answers(ctr, key, expect):
    out = S.philox4x32_10(*ctr, *key)
    assert tuple(int(x) for x in out) == expect


def test_philox_vectorised_equals_scalar():
    c0 = np.arange(64, dtype=np.uint32)
    vec = S.philox4x32_10(c0, 7, 9, 11, 123, 456)
    for i in (0, 5, 63):
        sc = S.philox4x32_10(i, 7, 9, 11, 123, 456)
        assert tuple(int(v[i]) for v in vec) == tuple(int(x) for x in sc)


def test_irwin_hall_extremes_and_moments():
    lo = S._irwin_hall4(np.array([0], np.uint32), np.array([0], np.uint32))[0]
    hi = S._irwin_hall4(np.array([0xFFFFFFFF], np.uint32), np.array([0xFFFFFFFF], np.uint32))[0]
    c = np.float32(math.sqrt(3.0 / (65536.0 ** 2 - 1)))
    assert lo == np.float32(-131070) * c and hi == np.float32(131070) * c
    ev, od = S.normal_pairs(np.arange(200000, dtype=np.uint32), 1, 2, 3, 42, 0)
    x = np.concatenate([ev, od]).astype(np.float64)
    assert abs(x.mean()) < 0.01 and abs(x.var() - 1.0) < 0.01
    # Irwin-Hall(4) excess kurtosis is -6/(5*4) = -0.3
    k = ((x - x.mean()) ** 4).mean() / x.var() ** 2 - 3.0
    assert abs(k + 0.3) < 0.03


def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.standard_normal(100000).astype(np.float32),
                        np.array([1.0, 1.00390625, 1.01171875, -2.5, 0.0, -0.0, 3.0e38], np.float32)])
    # ties: 1 + 2^-8 rounds to even (1.0); 1 + 3*2^-8 rounds up
    ours = S.bf16_rne_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(ours, ref)


def test_hidden_statistics_follow_the_ar1_field():
    w = S.TINY.with_(B=2, T=512, L=6, d=512)
    x = S.bf16_bits_to_f32(S.hidden(w)).astype(np.float64)
    assert abs(x.var() - 1.0) < 0.03
    ct = (x[:, 1:] * x[:, :-1]).mean()
    cl = (x[:, :, 1:] * x[:, :, :-1]).mean()
    cd = (x[:, 1:, 1:] * x[:, :-1, :-1]).mean()
    assert abs(ct - 0.9) < 0.02 and abs(cl - 0.8) < 0.02
    assert abs(cd - 0.72) < 0.02          # separable: rho_t * rho_l


def test_hidden_is_counter_based_per_stream_and_chunk_invariant():
    w = S.TINY.with_(T=40)
    full = S.hidden(w, seed=3)
    one = S.hidden_stream(3, 2, 40, w.L, w.d, w.rho_t, w.rho_l, t_chunk=7)
    assert np.array_equal(full[2], one)
    assert not np.array_equal(full[1], full[2])


def test_redraw_changes_only_the_redrawn_unit_and_its_successors():
    w = S.TINY.with_(T=12)
    att = np.zeros((w.T, w.L), np.uint8)
    base = S.hidden_stream(0, 0, w.T, w.L, w.d, w.rho_t, w.rho_l, att)
    att[5, 2] = 1
    re = S.hidden_stream(0, 0, w.T, w.L, w.d, w.rho_t, w.rho_l, att)
    diff = np.any(base != re, axis=-1)
    assert not diff[:5].any() and not diff[5, :2].any() and diff[5, 2]


def test_rho_l_one_makes_layers_identical():
    w = S.TINY.with_(T=8, rho_l=1.0)
    x = S.hidden(w)
    assert all(np.array_equal(x[:, :, 0], x[:, :, l]) for l in range(w.L))


def test_weights_scale_and_copy_init():
    w = S.TINY
    W = S.bf16_bits_to_f32(S.weights(w)).astype(np.float64)
    assert W.shape == (w.L, 3 * w.N, w.d)
    assert abs(W.var() * w.d - 1.0) < 0.03
    Wc = S.weights(w, copy_init=True)
    N = w.N
    for l in range(w.L):
        assert np.array_equal(Wc[l, N:2 * N], Wc[l, :N])
        assert np.array_equal(Wc[l, 2 * N:], Wc[(l + 1) % w.L, :N])


def test_workload_table():
    assert S.QWEN3_30B.units == 64 * 1024 * 48
    assert S.GPT_OSS_20B.expert_bytes == 49766400
    assert S.QWEN3_30B.expert_bytes == 9437184
