"""Failure detection on the GPU without a fault, and checkpoint / resume of
the state.  A bounded wait that runs out (a flag nothing sets; an mbarrier
phase nothing completes) latches CRC_ETIMEOUT in the state, the host reads it
through crc_state_read, the kernel has returned within about the wait limit,
and the context still runs the hot path correctly afterwards.  A state copied
to the host and restored elsewhere continues the streams exactly."""
import ctypes
import time

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


@pytest.mark.parametrize("kind", [0, 1], ids=["flag", "mbarrier"])
def test_expired_wait_reports_timeout_and_context_survives(C, kind):
    lib = C.load()
    w = S.QWEN3_30B.with_(B=2, T=140, L=2, d=128)
    p = C.problem_of(w)
    st = C.State(p)
    torch.cuda.synchronize()
    limit = 50_000_000                                   # 50 ms
    t0 = time.perf_counter()
    assert lib.crc_wait_probe(ctypes.byref(p), st.ptr, st.nbytes, kind, limit,
                              torch.cuda.current_stream().cuda_stream) == C.CRC_OK
    with pytest.raises(C.CrcError) as e:
        st.read()                                        # synchronises, reads the error word
    dt = time.perf_counter() - t0
    assert e.value.code == C.CRC_ETIMEOUT
    assert 0.05 <= dt < 1.5, dt
    assert C.crc_device_error() == C.CRC_OK
    # the context is intact: the fused step on a fresh state equals the two-kernel path
    Wd = C.synth_weights(w.L, w.N, w.d, seed=1)
    hd, _ = C.synth_hidden(w.B, w.T, w.L, w.d, seed=2)
    s1, s2 = C.State(p), C.State(p)
    ws = torch.empty(C.crc_fused_workspace_bytes(p), dtype=torch.uint8, device="cuda")
    C.route_and_cache(p, hd, Wd, s1, workspace=ws)
    C.cache_scan(p, C.route_scores(p, hd, Wd), s2)
    r1 = s1.read(want_caches=True)
    r2 = s2.read(want_caches=True)
    assert r1["error"] == 0 and r1["tokens"] == w.T
    assert (r1["cache_bits"] == r2["cache_bits"]).all() and r1["misses"] == r2["misses"]


def test_checkpoint_to_host_and_resume_elsewhere(C):
    """Checkpoint / resume: the state is position-independent bytes.  Copy it
    to the host after T1 tokens, restore it into a fresh buffer (another
    address), continue with the remaining tokens: the same final caches,
    counters and carried scores as one uninterrupted call."""
    w = S.QWEN3_30B.with_(B=2, T=300, L=3, d=128)
    p = C.problem_of(w)
    Wd = C.synth_weights(w.L, w.N, w.d, seed=7)
    hd, _ = C.synth_hidden(w.B, w.T, w.L, w.d, seed=8)
    ws = torch.empty(C.crc_fused_workspace_bytes(p), dtype=torch.uint8, device="cuda")
    whole = C.State(p)
    C.route_and_cache(p, hd, Wd, whole, workspace=ws)
    ref = whole.read(want_caches=True, want_retention=True, want_chain_counters=True)
    T1 = 170
    first = C.State(p)
    C.route_and_cache(p, hd[:, :T1].contiguous(), Wd, first, workspace=ws)
    saved = first.buf.cpu()                                # checkpoint
    del first
    resumed = C.State(p)
    resumed.buf.copy_(saved)                               # resume into a new buffer
    assert resumed.ptr != saved.data_ptr()
    C.route_and_cache(p, hd[:, T1:].contiguous(), Wd, resumed, workspace=ws)
    got = resumed.read(want_caches=True, want_retention=True, want_chain_counters=True)
    for k, v in ref.items():
        if hasattr(v, "shape"):
            assert (v == got[k]).all(), k
        else:
            assert v == got[k], k
