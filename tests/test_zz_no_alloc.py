"""The allocation-free entry point, crc_route_and_cache_noalloc.

It serves callers that cannot allocate device memory when they call in (a
serving framework that owns all device memory through its own pool, a
plug-in whose host forbids allocation after start-up): instead of a caller
workspace it uses a scratch array compiled into the library.  These tests
call it through the C ABI and check that two calls in a row, on different
inputs, give exactly what crc_route_and_cache gives -- in both layouts of the
array (the per-chunk router scores of the two-kernel path, and the fused
kernel's control words and ring of tiles) -- and that a problem too large for
the array is refused.  The file sorts last so that a run stopping
at its first failure has already run every other test.
"""
import ctypes

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


def _run(C, p, h, W, T, noalloc):
    st = C.State(p)
    tr = C.Trace.alloc(p, T)
    if noalloc:
        C.crc_route_and_cache_noalloc(p, h.data_ptr(), W.data_ptr(), T, st.ptr, st.nbytes, tr.c())
    else:
        ws = torch.empty(C.crc_workspace_bytes(p, T), dtype=torch.uint8, device="cuda")
        C.crc_route_and_cache(p, h.data_ptr(), W.data_ptr(), T, st.ptr, st.nbytes, tr.c(),
                              ws.data_ptr(), ws.numel())
    r = st.read(want_caches=True, want_retention=True, want_chain_counters=True)
    return r, tr


def test_noalloc_matches_route_and_cache_on_two_calls_in_a_row(C):
    # Qwen3-30B-shaped layers and streams: one token's scores take 4.7 MB, so the
    # 32 MiB array holds 7 tokens and the 40-token call runs in several chunks.
    w = S.QWEN3_30B.with_(T=40)
    p = C.problem_of(w)
    assert C.crc_workspace_bytes(p, 1) * 8 > C.NOALLOC_SCRATCH_BYTES
    W = C.synth_weights(w.L, w.N, w.d, seed=3)
    for call, seed in enumerate((21, 22)):           # two calls, different inputs
        h, _ = C.synth_hidden(w.B, w.T, w.L, w.d, seed=seed, rho_t=w.rho_t, rho_l=w.rho_l)
        ref, tref = _run(C, p, h, W, w.T, noalloc=False)
        got, tgot = _run(C, p, h, W, w.T, noalloc=True)
        assert got["error"] == 0 and got["tokens"] == w.T, call
        for k in ("cache_bits", "chain_counters"):
            assert np.array_equal(got[k], ref[k]), (call, k)
        assert np.array_equal(got["retention"].view(np.uint32), ref["retention"].view(np.uint32))
        assert torch.equal(tgot.topk, tref.topk), call
        assert torch.equal(tgot.misses, tref.misses), call
        assert torch.equal(tgot.proactive, tref.proactive), call


def test_noalloc_fused_kernel_in_the_scratch_on_two_calls_in_a_row(C):
    # A problem small enough for the fused kernel's ring to fit the array: an
    # untraced call (and one whose trace leaves out the rank-order Top-K) runs
    # the fused kernel with its control words and ring in the shared array.
    # Two calls in a row on different inputs, each against crc_route_and_cache
    # with a workspace of its own.
    w = S.QWEN3_30B.with_(B=8, L=6, T=300)
    p = C.problem_of(w)
    assert 0 < C.crc_fused_workspace_bytes(p) <= C.NOALLOC_SCRATCH_BYTES
    W = C.synth_weights(w.L, w.N, w.d, seed=4)
    ws = torch.empty(C.crc_fused_workspace_bytes(p), dtype=torch.uint8, device="cuda")
    for call, seed in enumerate((23, 24)):
        h, _ = C.synth_hidden(w.B, w.T, w.L, w.d, seed=seed, rho_t=w.rho_t, rho_l=w.rho_l)
        ref_st = C.State(p)
        C.crc_route_and_cache(p, h.data_ptr(), W.data_ptr(), w.T, ref_st.ptr, ref_st.nbytes,
                              None, ws.data_ptr(), ws.numel())
        ref = ref_st.read(want_caches=True, want_retention=True, want_chain_counters=True)
        for traced in (False, True):
            st = C.State(p)
            tr = C.Trace.alloc(p, w.T, rank_order=False, topk_set=True) if traced else None
            C.crc_profile_begin()
            C.crc_route_and_cache_noalloc(p, h.data_ptr(), W.data_ptr(), w.T, st.ptr, st.nbytes,
                                          None if tr is None else tr.c())
            kt = C.crc_profile_end()
            assert kt["fused"]["launches"] == 1 and kt["router"]["launches"] == 0, (call, traced)
            got = st.read(want_caches=True, want_retention=True, want_chain_counters=True)
            assert got["error"] == 0 and got["tokens"] == w.T, (call, traced)
            for k in ("cache_bits", "chain_counters"):
                assert np.array_equal(got[k], ref[k]), (call, traced, k)
            assert np.array_equal(got["retention"].view(np.uint32),
                                  ref["retention"].view(np.uint32)), (call, traced)


def test_noalloc_refuses_problems_larger_than_its_scratch(C):
    # 512 streams x 94 layers x 384 scores x 4 bytes = 74 MB for a single token
    w = S.LARGE
    p = C.problem_of(w)
    assert C.crc_workspace_bytes(p, 1) > C.NOALLOC_SCRATCH_BYTES
    rc = C.load().crc_route_and_cache_noalloc(ctypes.byref(p), 256, 256, 4, 256,
                                              C.crc_state_bytes(p), None, None)
    assert rc == C.CRC_EUNSUPPORTED
