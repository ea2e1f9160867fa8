"""Host-only checks of the C-ABI library: it builds, loads, exports every
symbol include/crc.h declares, and rejects bad arguments before touching the
GPU (no compute call is made here)."""
import ctypes
import os
import re

import pytest

import crc_synth as S

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def crc():
    from paper_2609_04895_gb300 import build
    build.build()
    from paper_2609_04895_gb300 import crc as C
    C.load()
    return C


def header_functions():
    src = open(os.path.join(ROOT, "include", "crc.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(crc_[a-z_]+)\s*\(", src)))


def test_every_declared_symbol_is_exported_and_bound(crc):
    names = header_functions()
    assert len(names) >= 12
    lib = crc.load()
    bound = {n for n, _, _ in crc.EXPORTS}
    for n in names:
        assert hasattr(lib, n), n
        assert n in bound, n


def test_struct_layouts_match_header(crc):
    assert ctypes.sizeof(crc.crc_problem) == 40
    assert ctypes.sizeof(crc.crc_trace) == 48
    assert ctypes.sizeof(crc.crc_transfer) == 24
    assert ctypes.sizeof(crc.crc_stats) == 56


def test_sizes(crc):
    p = crc.problem_of(S.QWEN3_30B)
    B, L, N = p.B, p.L, p.N
    # header, chains, retention, p^S carry, a comparison policy's integer priorities
    expect = 256 + B * L * 64 + B * L * N * 4 + 2 * B * N * 4 + B * L * N * 4
    assert crc.crc_state_bytes(p) == (expect + 255) // 256 * 256
    assert crc.crc_workspace_bytes(p, 16) == B * 16 * L * 3 * N * 4
    assert crc.crc_workspace_bytes(p, 0) == 0


@pytest.mark.parametrize("field,value,code", [
    ("C", 4, 2),        # C < K
    ("C", 200, 2),      # C > N
    ("N", 40, 2),       # N % 16 != 0
    ("K", 40, 2),       # K > 32
    ("R", 129, 2),      # R > N
    ("L", 0, 1),
    ("B", 0, 1),
    ("reserved", 1, 1),
])
def test_problem_validation(crc, field, value, code):
    p = crc.problem_of(S.QWEN3_30B)
    setattr(p, field, value)
    assert crc.crc_state_bytes(p) == 0
    lib = crc.load()
    assert lib.crc_state_init(ctypes.byref(p), None, 0, None) == code
    assert lib.crc_route_scores(ctypes.byref(p), 16, 16, 1, 3, 16, None) == code


def test_router_limits_and_pointer_checks(crc):
    lib = crc.load()
    p = crc.problem_of(S.QWEN3_30B.with_(N=256, C=32))
    assert crc.crc_state_bytes(p) > 0                       # the scan takes N = 256
    assert lib.crc_route_scores(ctypes.byref(p), 16, 16, 1, 3, 16, None) == crc.CRC_EUNSUPPORTED
    p = crc.problem_of(S.QWEN3_30B)
    assert lib.crc_route_scores(ctypes.byref(p), 16, 16, 0, 3, 16, None) == crc.CRC_OK   # T = 0
    assert lib.crc_route_scores(ctypes.byref(p), None, 16, 4, 3, 16, None) == crc.CRC_EINVAL
    assert lib.crc_route_scores(ctypes.byref(p), 8, 16, 4, 3, 16, None) == crc.CRC_EINVAL
    assert lib.crc_route_scores(ctypes.byref(p), 16, 16, 4, 4, 16, None) == crc.CRC_EINVAL
    assert lib.crc_route_scores(ctypes.byref(p), 16, 16, -1, 3, 16, None) == crc.CRC_EINVAL
    n = crc.crc_state_bytes(p)
    assert lib.crc_cache_scan(ctypes.byref(p), 16, 4, 256, n - 256, None, None) == crc.CRC_ESTATE
    assert lib.crc_cache_scan(ctypes.byref(p), 16, 4, 128, n, None, None) == crc.CRC_EINVAL
    ws = crc.crc_workspace_bytes(p, 1)
    assert lib.crc_route_and_cache(ctypes.byref(p), 16, 16, 4, 256, n, None, 256, ws - 1,
                                   None) == crc.CRC_EINVAL
    assert lib.crc_synth_hidden(1, 1, 1, 3, 0, 0, 0.5, 0.5, None, 16, 16, None) == crc.CRC_EINVAL
    assert lib.crc_synth_hidden(1, 1, 1, 4, 0, 0, 1.5, 0.5, None, 16, 16, None) == crc.CRC_EINVAL


def test_host_input_call_argument_checks(crc):
    """crc_route_and_cache_host refuses bad arguments before it touches the GPU."""
    lib = crc.load()
    p = crc.problem_of(S.QWEN3_30B)
    half = p.B * 128 * p.L * p.d * 2
    assert crc.crc_host_staging_bytes(p, 128) == 2 * ((half + 255) // 256 * 256)
    assert crc.crc_host_staging_bytes(p, 0) == 0
    n = crc.crc_state_bytes(p)
    sb = crc.crc_host_staging_bytes(p, 64)
    ws = crc.crc_fused_workspace_bytes(p)
    call = lambda h, T, chunk, stg, stg_bytes: lib.crc_route_and_cache_host(   # noqa: E731
        ctypes.byref(p), h, 16, T, chunk, 256, n, stg, stg_bytes, 256, ws, None)
    assert call(16, 0, 64, 256, sb) == crc.CRC_OK                  # T = 0: nothing queued
    assert call(16, -1, 64, 256, sb) == crc.CRC_EINVAL
    assert call(16, 128, 0, 256, sb) == crc.CRC_EINVAL             # chunk < 1
    assert call(None, 128, 64, 256, sb) == crc.CRC_EINVAL          # no host buffer
    assert call(8, 128, 64, 256, sb) == crc.CRC_EINVAL             # host buffer misaligned
    assert call(16, 128, 64, 128, sb) == crc.CRC_EINVAL            # staging misaligned
    assert call(16, 128, 64, 256, sb - 1) == crc.CRC_EINVAL        # staging too small
    assert call(16, 128, 128, 256, sb) == crc.CRC_EINVAL           # ... for 128-token chunks
    assert lib.crc_route_and_cache_host(ctypes.byref(p), 16, 16, 128, 64, 256, n - 256, 256, sb,
                                        256, ws, None) == crc.CRC_ESTATE


def test_host_alloc_argument_checks(crc):
    lib = crc.load()
    out = ctypes.c_void_p(1)
    assert lib.crc_host_alloc(0, ctypes.byref(out)) == crc.CRC_EINVAL and not out.value
    assert lib.crc_host_alloc(64, None) == crc.CRC_EINVAL
    assert lib.crc_host_free(None) == crc.CRC_OK
    assert lib.crc_host_free(4096) == crc.CRC_EINVAL         # not handed out by the library
    assert "host memory" in crc.crc_strerror(crc.CRC_ENOMEM)


def test_wait_probe_argument_checks(crc):
    lib = crc.load()
    p = crc.problem_of(S.TINY)
    n = crc.crc_state_bytes(p)
    assert lib.crc_wait_probe(ctypes.byref(p), None, n, 0, 10**7, None) == crc.CRC_EINVAL
    assert lib.crc_wait_probe(ctypes.byref(p), 128, n, 0, 10**7, None) == crc.CRC_EINVAL
    assert lib.crc_wait_probe(ctypes.byref(p), 256, n, 2, 10**7, None) == crc.CRC_EINVAL
    assert lib.crc_wait_probe(ctypes.byref(p), 256, n - 1, 0, 10**7, None) == crc.CRC_EINVAL


def test_policy_scan_argument_checks(crc):
    lib = crc.load()
    p = crc.problem_of(S.QWEN3_30B)
    n = crc.crc_state_bytes(p)
    scan = lambda policy, lam, T=4, scores=16: lib.crc_cache_scan_policy(   # noqa: E731
        ctypes.byref(p), scores, T, 256, n, None, policy, lam, None)
    assert scan(0, 1) == crc.CRC_EINVAL                     # the method itself: crc_cache_scan
    assert scan(5, 1) == crc.CRC_EINVAL
    assert scan(crc.POLICIES["lrfu"], -1) == crc.CRC_EINVAL
    assert scan(crc.POLICIES["lrfu"], 9) == crc.CRC_EINVAL
    assert scan(crc.POLICIES["lru"], 1, T=-1) == crc.CRC_EINVAL
    assert scan(crc.POLICIES["lru"], 1, T=0) == crc.CRC_OK
    assert scan(crc.POLICIES["lfu"], 1, scores=8) == crc.CRC_EINVAL
    assert lib.crc_cache_scan_policy(ctypes.byref(p), 16, 4, 256, n - 256, None, 1, 1,
                                     None) == crc.CRC_ESTATE
    assert lib.crc_state_read_aux(ctypes.byref(p), 256, n, None, None) == crc.CRC_EINVAL


def test_cache_loss_argument_checks(crc):
    lib = crc.load()
    p = crc.problem_of(S.QWEN3_30B)
    # per-task fp64 sums: B * L tasks per token chunk, 16 chunks of 64 tokens at T = 1024
    assert crc.crc_loss_workspace_bytes(p, 1024) == 64 * 48 * 16 * 16
    assert crc.crc_loss_workspace_bytes(p, 0) == 0
    # N <= 32: chunks are sized at launch, so one slot per stream, layer and 32 tokens
    g = crc.problem_of(S.GPT_OSS_20B)
    assert crc.crc_loss_workspace_bytes(g, 2048) == 128 * 24 * 64 * 16
    assert crc.crc_loss_workspace_bytes(g, 33) == 128 * 24 * 2 * 16
    ws = crc.crc_loss_workspace_bytes(p, 8)
    call = lambda T=8, heads=3, top_b=20, tau=0.03, wT=1.0, wST=1.0, probs=256, loss=256, \
        means=None, grad=None, ws_ptr=256, ws_bytes=ws: lib.crc_cache_loss(  # noqa: E731
            ctypes.byref(p), probs, T, heads, top_b, tau, wT, wST, loss, means, grad, ws_ptr,
            ws_bytes, None)
    assert call(T=0) == crc.CRC_OK
    assert call(T=-1) == crc.CRC_EINVAL
    assert call(heads=1) == crc.CRC_EINVAL
    assert call(top_b=0) == crc.CRC_EINVAL and call(top_b=129) == crc.CRC_EINVAL
    assert call(tau=0.0) == crc.CRC_EINVAL and call(tau=float("nan")) == crc.CRC_EINVAL
    assert call(tau=1e-320) == crc.CRC_EINVAL                 # 1 / tau overflows
    assert call(wT=float("inf")) == crc.CRC_EINVAL
    assert call(probs=None) == crc.CRC_EINVAL and call(probs=8) == crc.CRC_EINVAL
    assert call(grad=256) == crc.CRC_EINVAL                   # aliases probs
    assert call(grad=4104) == crc.CRC_EINVAL                  # misaligned
    assert call(means=512, ws_bytes=ws - 1) == crc.CRC_EINVAL
    assert call(means=512, ws_ptr=None) == crc.CRC_EINVAL
    assert call(means=512, ws_ptr=128) == crc.CRC_EINVAL
    assert call(loss=None) == crc.CRC_OK                      # nothing requested


def test_strerror(crc):
    assert "unsupported" in crc.crc_strerror(2) or "limits" in crc.crc_strerror(2)
    assert crc.crc_strerror(99) == "unknown error code"


def test_product_fails_loudly_without_library(tmp_path):
    from paper_2609_04895_gb300 import crc as C
    saved = C._lib
    try:
        C._lib = None
        with pytest.raises(ImportError):
            C.load(str(tmp_path / "missing.so"))
    finally:
        C._lib = saved


def test_product_never_imports_the_oracle():
    pkg = os.path.join(ROOT, "paper_2609_04895_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h")):
                txt = open(os.path.join(dirpath, f)).read()
                assert "import oracle" not in txt and "from oracle" not in txt, f
                assert "crc_oracle" not in txt, f
