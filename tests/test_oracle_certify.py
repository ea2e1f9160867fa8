"""The margin-certifying walk of ``oracle.certify`` (no GPU).

Its accepted draws must be the generator's own field under the re-draw
table it reports, and its per-access trace must be what the whole-sequence
fp64 oracle computes on those hidden states -- the walk is the oracle run
unit by unit, not a second implementation of it -- with every certified
unit's margin at or above the tolerance.
"""
import numpy as np
import pytest

import crc_synth as S


@pytest.mark.parametrize("w", [S.TINY, S.TINY.with_(L=1, T=96, R=2),
                               S.GPT_OSS_20B.with_(B=2, T=24, L=3, d=256)],
                         ids=["tiny", "one-layer", "gptoss-small"])
def test_walk_equals_generator_and_whole_sequence_oracle(oracle_lib, w):
    from oracle import certify
    W = S.weights(w, seed=12)
    streams = list(range(w.B))
    r = certify.certified_streams(w, W, 11, streams, processes=1)
    assert r["certified"].all()
    assert int(r["redraws"].sum()) > 0                 # the repair was exercised
    for i, b in enumerate(streams):
        ref = S.hidden_stream(11, b, w.T, w.L, w.d, w.rho_t, w.rho_l, attempts=r["attempts"][i])
        assert np.array_equal(ref, r["hidden"][i])
    o = oracle_lib.run(r["hidden"], W, w.N, w.K, w.C, w.R)
    for k in ("topk", "misses", "proactive", "cache_bits", "counters", "margins"):
        assert np.array_equal(o[k], r[k]), k
    assert np.array_equal(o["aT"], r["aT"])
    assert o["margins"].min() >= 1e-3


def test_walk_without_redraws_flags_the_close_units(oracle_lib):
    # max_tries = 1 keeps every first draw: the flags are then exactly the
    # units the whole-sequence oracle finds closer than the tolerance
    from oracle import certify
    w = S.TINY.with_(T=128)
    W = S.weights(w, seed=2)
    r = certify.certified_streams(w, W, 3, range(w.B), max_tries=1, processes=1)
    assert not r["attempts"].any()
    o = oracle_lib.run(S.hidden(w, seed=3), W, w.N, w.K, w.C, w.R)
    assert np.array_equal(~r["certified"], o["margins"] < 1e-3)
    assert (~r["certified"]).any()


def test_process_pool_equals_in_process(oracle_lib):
    from oracle import certify
    w = S.TINY.with_(T=48)
    W = S.weights(w, seed=5)
    a = certify.certified_streams(w, W, 6, [0, 3], processes=1)
    b = certify.certified_streams(w, W, 6, [0, 3], processes=2)
    for k in a:
        assert np.array_equal(a[k], b[k]), k
