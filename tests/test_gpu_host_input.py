"""crc_route_and_cache_host (hidden states in host memory, chunked copies
overlapped with the step) against crc_route_and_cache on the same hidden
states already on the device: counters, cache sets, carried retention scores
and token count bit for bit, over ragged chunkings, both fused kernels (CTA
pairs for N = 128, one CTA per tile for N = 32), the two-kernel path (small
workspace), pageable host memory, and host rows longer than the largest 2-D
copy pitch (one copy per stream instead of one 2-D copy).  Also the pinned
huge-page host allocator (crc_host_alloc / crc_host_free) behind
pinned_empty."""
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


def final(C, st):
    r = st.read(want_caches=True, want_retention=True, want_chain_counters=True)
    assert r["error"] == 0
    return r


def same(r1, r2):
    for k, v in r1.items():
        if isinstance(v, np.ndarray):
            assert np.array_equal(v, r2[k]), k
        else:
            assert v == r2[k], k


def run_pair(C, w, T, chunk, pinned=True, small_ws=False, seed=5):
    p = C.problem_of(w)
    Wd = C.synth_weights(w.L, w.N, w.d, seed=seed)
    hd, _ = C.synth_hidden(w.B, T, w.L, w.d, seed=seed + 1)
    ws_bytes = C.crc_workspace_bytes(p, 16) if small_ws else C.crc_fused_workspace_bytes(p)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device="cuda")
    st1, st2 = C.State(p), C.State(p)
    C.crc_route_and_cache(p, hd.data_ptr(), Wd.data_ptr(), T, st1.ptr, st1.nbytes, None,
                          ws.data_ptr(), ws.numel(), None)
    ref = final(C, st1)
    h_host = C.pinned_empty(hd.shape, hd.dtype) if pinned else torch.empty(hd.shape,
                                                                           dtype=hd.dtype)
    h_host.copy_(hd)
    torch.cuda.synchronize()
    del hd
    C.route_and_cache_host(p, h_host, Wd, st2, chunk_tokens=chunk, workspace=ws)
    got = final(C, st2)
    same(ref, got)
    return ref


CASES = [
    ("pairs-ragged", S.QWEN3_30B.with_(B=4, L=3, d=256), 300, 128),
    ("pairs-one-chunk", S.QWEN3_30B.with_(B=2, L=2, d=128), 150, 512),
    ("pairs-small-chunks", S.QWEN3_30B.with_(B=2, L=2, d=128), 97, 16),
    ("n32-ragged", S.GPT_OSS_20B.with_(B=3, L=2, d=2880), 200, 64),
    ("n16-r0", S.TINY.with_(B=5, R=0), 130, 48),
]


@pytest.mark.parametrize("name,w,T,chunk", CASES, ids=[c[0] for c in CASES])
def test_host_call_equals_device_call(C, name, w, T, chunk):
    r = run_pair(C, w, T, chunk)
    assert r["tokens"] == T and r["accesses"] == w.B * T * w.L * w.K


def test_pageable_host_memory(C):
    run_pair(C, S.QWEN3_30B.with_(B=2, L=2, d=128), 140, 64, pinned=False)


def test_two_kernel_path_through_host_call(C):
    run_pair(C, S.QWEN3_30B.with_(B=2, L=2, d=128), 70, 32, small_ws=True)


def test_rows_beyond_the_2d_copy_pitch(C):
    """One stream's T tokens longer than the device's largest 2-D copy pitch:
    the call copies stream by stream."""
    lib = ctypes.CDLL("libcuda.so.1")
    assert lib.cuInit(0) == 0
    dev, pitch = ctypes.c_int(), ctypes.c_int()
    assert lib.cuDeviceGet(ctypes.byref(dev), torch.cuda.current_device()) == 0
    assert lib.cuDeviceGetAttribute(ctypes.byref(pitch), 11, dev) == 0    # MAX_PITCH
    w = S.TINY.with_(B=2, L=8, d=1024, N=16, K=2, C=4, R=1)
    row = w.L * w.d * 2
    T = pitch.value // row + 1
    if 2 * T * row > (6 << 30):
        pytest.skip(f"max pitch {pitch.value} needs {2 * T * row} host bytes")
    run_pair(C, w, T, 4096)


def test_pinned_huge_page_allocator(C):
    t = C.pinned_empty((3000, 77), torch.float32)
    assert t.is_pinned() and t.data_ptr() % 65536 == 0
    x = torch.randn(3000, 77)
    t.copy_(x)
    d = t.cuda(non_blocking=True)
    back = C.pinned_empty((3000, 77), torch.float32)
    back.copy_(d, non_blocking=True)
    torch.cuda.synchronize()
    assert torch.equal(back, x)
    view = t[10:20]
    del t                                  # the mapping lives while a view does
    assert torch.equal(view, x[10:20])
    del view, back
    lib = C.load()
    ptr = ctypes.c_void_p()
    assert lib.crc_host_alloc(1 << 20, ctypes.byref(ptr)) == C.CRC_OK and ptr.value
    assert lib.crc_host_free(ptr) == C.CRC_OK
    assert lib.crc_host_free(ptr) == C.CRC_EINVAL          # already released
