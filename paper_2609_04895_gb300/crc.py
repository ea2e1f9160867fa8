"""ctypes binding of the CUDA library (include/crc.h), names as in the C ABI.

Argument marshalling only: every step of the routing and cache path runs in
the library's kernels.  PyTorch supplies device memory and streams.  There
is no fallback: if libcrc.so is missing or a call fails, an exception is
raised.
"""
from __future__ import annotations

import ctypes
import math
import os
import threading
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libcrc.so")

(CRC_OK, CRC_EINVAL, CRC_EUNSUPPORTED, CRC_ECUDA, CRC_ETIMEOUT, CRC_ESTATE, CRC_EDEVICE,
 CRC_ENOMEM) = range(8)


class crc_problem(ctypes.Structure):
    _fields_ = [("L", ctypes.c_int32), ("N", ctypes.c_int32), ("K", ctypes.c_int32),
                ("d", ctypes.c_int32), ("C", ctypes.c_int32), ("R", ctypes.c_int32),
                ("B", ctypes.c_int32), ("reserved", ctypes.c_int32),
                ("expert_bytes", ctypes.c_uint64)]


class crc_trace(ctypes.Structure):
    _fields_ = [("topk_dev", ctypes.c_void_p), ("misses_dev", ctypes.c_void_p),
                ("proactive_dev", ctypes.c_void_p), ("cache_mid_dev", ctypes.c_void_p),
                ("cache_after_dev", ctypes.c_void_p), ("topk_set_dev", ctypes.c_void_p)]


class crc_transfer(ctypes.Structure):
    _fields_ = [("t", ctypes.c_int32), ("l", ctypes.c_int32), ("expert", ctypes.c_int32),
                ("slot", ctypes.c_int32), ("evicted", ctypes.c_int32),
                ("proactive", ctypes.c_int32)]


TRANSFER_DTYPE = np.dtype([("t", np.int32), ("l", np.int32), ("expert", np.int32),
                           ("slot", np.int32), ("evicted", np.int32), ("proactive", np.int32)])


class crc_stats(ctypes.Structure):
    _fields_ = [("accesses", ctypes.c_uint64), ("hits", ctypes.c_uint64),
                ("misses", ctypes.c_uint64), ("proactive", ctypes.c_uint64),
                ("traffic_bytes", ctypes.c_uint64), ("tokens", ctypes.c_uint64),
                ("error", ctypes.c_uint32), ("reserved", ctypes.c_uint32)]


class crc_report(ctypes.Structure):
    _fields_ = [("hit", ctypes.c_double), ("adj_hit", ctypes.c_double),
                ("traffic_bytes", ctypes.c_double), ("load_per_token_bytes", ctypes.c_double)]


KERNEL_KINDS = {"router": 0, "scan": 1, "state": 2, "synth": 3, "fused": 4, "loss": 5,
                "loss_means": 6}


class crc_kernel_times(ctypes.Structure):
    _fields_ = [("launches", ctypes.c_uint64 * 8), ("ms", ctypes.c_double * 8)]


class CrcError(RuntimeError):
    def __init__(self, code: int, what: str):
        self.code = code
        super().__init__(f"{what}: {crc_strerror(code)} (code {code})")


_lib = None
_lock = threading.Lock()

# (name, restype, argtypes) of every exported symbol
P, I32, U32, U64, SZ, D = (ctypes.c_void_p, ctypes.c_int32, ctypes.c_uint32, ctypes.c_uint64,
                           ctypes.c_size_t, ctypes.c_double)
PP = ctypes.POINTER(crc_problem)
EXPORTS = [
    ("crc_state_bytes", SZ, [PP]),
    ("crc_state_init", ctypes.c_int, [PP, P, SZ, P]),
    ("crc_state_read", ctypes.c_int, [PP, P, SZ, ctypes.POINTER(crc_stats), P, P, P, P]),
    ("crc_route_scores", ctypes.c_int, [PP, P, P, I32, I32, P, P]),
    ("crc_cache_scan", ctypes.c_int, [PP, P, I32, P, SZ, ctypes.POINTER(crc_trace), P]),
    ("crc_workspace_bytes", SZ, [PP, I32]),
    ("crc_fused_workspace_bytes", SZ, [PP]),
    ("crc_route_and_cache", ctypes.c_int,
     [PP, P, P, I32, P, SZ, ctypes.POINTER(crc_trace), P, SZ, P]),
    ("crc_route_and_cache_noalloc", ctypes.c_int,
     [PP, P, P, I32, P, SZ, ctypes.POINTER(crc_trace), P]),
    ("crc_host_staging_bytes", SZ, [PP, I32]),
    ("crc_host_alloc", ctypes.c_int, [SZ, ctypes.POINTER(ctypes.c_void_p)]),
    ("crc_host_free", ctypes.c_int, [P]),
    ("crc_wait_probe", ctypes.c_int, [PP, P, SZ, I32, U64, P]),
    ("crc_route_and_cache_host", ctypes.c_int, [PP, P, P, I32, I32, P, SZ, P, SZ, P, SZ, P]),
    ("crc_device_error", ctypes.c_int, []),
    ("crc_cache_scan_policy", ctypes.c_int,
     [PP, P, I32, P, SZ, ctypes.POINTER(crc_trace), I32, I32, P]),
    ("crc_state_read_aux", ctypes.c_int, [PP, P, SZ, P, P]),
    ("crc_loss_workspace_bytes", SZ, [PP, I32]),
    ("crc_transfer_plan", ctypes.c_int, [PP, I32, P, P, P, P, P, ctypes.c_int64, P]),
    ("crc_transfer_replay", ctypes.c_int, [PP, P, ctypes.c_int64, P, ctypes.c_int64, P, P]),
    ("crc_cache_loss", ctypes.c_int, [PP, P, I32, I32, I32, D, D, D, P, P, P, P, SZ, P]),
    ("crc_metrics", ctypes.c_int, [PP, ctypes.POINTER(crc_stats), ctypes.POINTER(crc_report)]),
    ("crc_load_time", ctypes.c_int, [PP, ctypes.POINTER(crc_stats), D, D,
                                      ctypes.POINTER(ctypes.c_double)]),
    ("crc_launch_count", U64, []),
    ("crc_strerror", ctypes.c_char_p, [ctypes.c_int]),
    ("crc_profile_begin", ctypes.c_int, []),
    ("crc_profile_end", ctypes.c_int, [ctypes.POINTER(crc_kernel_times)]),
    ("crc_synth_hidden", ctypes.c_int, [I32, I32, I32, I32, I32, U32, D, D, P, P, P, P]),
    ("crc_synth_weights", ctypes.c_int, [I32, I32, I32, U32, I32, P, P]),
]


def load(path: str = LIB_PATH):
    """Load libcrc.so (built by paper_2609_04895_gb300.build); raises if absent."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(path):
                raise ImportError(
                    f"CUDA library not built: {path} (run paper_2609_04895_gb300.build.build())")
            lib = ctypes.CDLL(path)
            for name, res, args in EXPORTS:
                f = getattr(lib, name)
                f.restype = res
                f.argtypes = args
            _lib = lib
    return _lib


def _ck(rc: int, what: str):
    if rc != CRC_OK:
        raise CrcError(rc, what)


def _stream(stream) -> int:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _ptr(t) -> int:
    if t is None:
        return None
    return t.data_ptr()


# --------------------------------------------------------------------------- #
# C-ABI names
# --------------------------------------------------------------------------- #
def crc_strerror(code: int) -> str:
    try:
        return load().crc_strerror(code).decode()
    except ImportError:
        return f"error {code}"


def crc_state_bytes(p: crc_problem) -> int:
    return int(load().crc_state_bytes(ctypes.byref(p)))


def crc_state_init(p: crc_problem, state_ptr: int, state_bytes: int, stream=None):
    _ck(load().crc_state_init(ctypes.byref(p), state_ptr, state_bytes, _stream(stream)),
        "crc_state_init")


def crc_state_read(p: crc_problem, state_ptr: int, state_bytes: int, stream=None,
                   want_caches: bool = False, want_retention: bool = False,
                   want_chain_counters: bool = False) -> dict:
    st = crc_stats()
    B, L, N = p.B, p.L, p.N
    bits = np.zeros((B, L, (N + 31) // 32), np.uint32) if want_caches else None
    ret = np.zeros((B, L, N), np.float32) if want_retention else None
    cc = np.zeros((B, L, 3), np.uint64) if want_chain_counters else None
    rc = load().crc_state_read(ctypes.byref(p), state_ptr, state_bytes, ctypes.byref(st),
                               None if bits is None else bits.ctypes.data,
                               None if ret is None else ret.ctypes.data,
                               None if cc is None else cc.ctypes.data, _stream(stream))
    _ck(rc, "crc_state_read")
    out = {f: int(getattr(st, f)) for f, _ in crc_stats._fields_ if f != "reserved"}
    out.update(cache_bits=bits, retention=ret, chain_counters=cc)
    return out


def crc_route_scores(p: crc_problem, hidden_ptr: int, w_ptr: int, T: int, heads: int,
                     scores_ptr: int, stream=None):
    _ck(load().crc_route_scores(ctypes.byref(p), hidden_ptr, w_ptr, T, heads, scores_ptr,
                                _stream(stream)), "crc_route_scores")


def crc_cache_scan(p: crc_problem, scores_ptr: int, T: int, state_ptr: int, state_bytes: int,
                   trace: crc_trace | None = None, stream=None):
    _ck(load().crc_cache_scan(ctypes.byref(p), scores_ptr, T, state_ptr, state_bytes,
                              None if trace is None else ctypes.byref(trace), _stream(stream)),
        "crc_cache_scan")


# comparison policies (crc.h CRC_POLICY_*)
POLICIES = {"lru": 1, "lfu": 2, "lrfu": 3, "spatio_lru": 4}


def crc_cache_scan_policy(p: crc_problem, scores_ptr: int, T: int, state_ptr: int,
                          state_bytes: int, trace: crc_trace | None, policy: int,
                          lambda_halves: int = 1, stream=None):
    _ck(load().crc_cache_scan_policy(ctypes.byref(p), scores_ptr, T, state_ptr, state_bytes,
                                     None if trace is None else ctypes.byref(trace), policy,
                                     lambda_halves, _stream(stream)),
        "crc_cache_scan_policy")


def crc_state_read_aux(p: crc_problem, state_ptr: int, state_bytes: int,
                       stream=None) -> np.ndarray:
    aux = np.zeros((p.B, p.L, p.N), np.uint32)
    _ck(load().crc_state_read_aux(ctypes.byref(p), state_ptr, state_bytes, aux.ctypes.data,
                                  _stream(stream)), "crc_state_read_aux")
    return aux


def crc_loss_workspace_bytes(p: crc_problem, T: int) -> int:
    return int(load().crc_loss_workspace_bytes(ctypes.byref(p), T))


def crc_cache_loss(p: crc_problem, probs_ptr: int, T: int, heads: int, top_b: int, tau: float,
                   w_T: float, w_ST: float, loss_ptr, means_ptr, grad_ptr, ws_ptr, ws_bytes: int,
                   stream=None):
    _ck(load().crc_cache_loss(ctypes.byref(p), probs_ptr, T, heads, top_b, tau, w_T, w_ST,
                              loss_ptr, means_ptr, grad_ptr, ws_ptr, ws_bytes, _stream(stream)),
        "crc_cache_loss")


def crc_transfer_plan(p: crc_problem, T: int, mid_ptr, after_ptr, start_ptr, slot_expert_ptr,
                      out_ptr, max_out: int) -> int:
    n = ctypes.c_int64(0)
    _ck(load().crc_transfer_plan(ctypes.byref(p), T, mid_ptr, after_ptr, start_ptr,
                                 slot_expert_ptr, out_ptr, max_out, ctypes.byref(n)),
        "crc_transfer_plan")
    return int(n.value)


def crc_transfer_replay(p: crc_problem, plan_ptr, n: int, pool_ptr, pool_experts: int,
                        slots_ptr, stream=None):
    _ck(load().crc_transfer_replay(ctypes.byref(p), plan_ptr, n, pool_ptr, pool_experts,
                                   slots_ptr, _stream(stream)), "crc_transfer_replay")


def crc_workspace_bytes(p: crc_problem, chunk_tokens: int) -> int:
    return int(load().crc_workspace_bytes(ctypes.byref(p), chunk_tokens))


def crc_fused_workspace_bytes(p: crc_problem) -> int:
    return int(load().crc_fused_workspace_bytes(ctypes.byref(p)))


def crc_route_and_cache(p: crc_problem, hidden_ptr: int, w_ptr: int, T: int, state_ptr: int,
                        state_bytes: int, trace: crc_trace | None, ws_ptr: int, ws_bytes: int,
                        stream=None):
    _ck(load().crc_route_and_cache(ctypes.byref(p), hidden_ptr, w_ptr, T, state_ptr, state_bytes,
                                   None if trace is None else ctypes.byref(trace), ws_ptr,
                                   ws_bytes, _stream(stream)), "crc_route_and_cache")


def pinned_empty(shape, dtype):
    """A host tensor in pinned huge-page memory from crc_host_alloc, released
    with crc_host_free when the tensor (and every view of it) is gone."""
    import torch
    nbytes = math.prod(shape) * torch.empty((), dtype=dtype).element_size()
    ptr = ctypes.c_void_p()
    _ck(load().crc_host_alloc(max(nbytes, 1), ctypes.byref(ptr)), "crc_host_alloc")
    addr = ptr.value
    lib = load()

    class _Pinned(ctypes.c_uint8 * max(nbytes, 1)):
        def __del__(self):
            lib.crc_host_free(addr)

    buf = _Pinned.from_address(addr)
    return torch.frombuffer(buf, dtype=torch.uint8)[:nbytes].view(dtype).view(shape)


def crc_host_staging_bytes(p: crc_problem, chunk_tokens: int) -> int:
    return int(load().crc_host_staging_bytes(ctypes.byref(p), chunk_tokens))


def crc_route_and_cache_host(p: crc_problem, hidden_host_ptr: int, w_ptr: int, T: int,
                             chunk_tokens: int, state_ptr: int, state_bytes: int,
                             staging_ptr: int, staging_bytes: int, ws_ptr: int, ws_bytes: int,
                             stream=None):
    _ck(load().crc_route_and_cache_host(ctypes.byref(p), hidden_host_ptr, w_ptr, T, chunk_tokens,
                                        state_ptr, state_bytes, staging_ptr, staging_bytes,
                                        ws_ptr, ws_bytes, _stream(stream)),
        "crc_route_and_cache_host")


NOALLOC_SCRATCH_BYTES = 32 << 20


def crc_route_and_cache_noalloc(p: crc_problem, hidden_ptr: int, w_ptr: int, T: int,
                                state_ptr: int, state_bytes: int, trace: crc_trace | None = None,
                                stream=None):
    """crc_route_and_cache using the library's built-in scratch array (no workspace)."""
    _ck(load().crc_route_and_cache_noalloc(ctypes.byref(p), hidden_ptr, w_ptr, T, state_ptr,
                                           state_bytes,
                                           None if trace is None else ctypes.byref(trace),
                                           _stream(stream)), "crc_route_and_cache_noalloc")


def crc_device_error() -> int:
    return int(load().crc_device_error())


def crc_launch_count() -> int:
    return int(load().crc_launch_count())


def crc_profile_begin():
    _ck(load().crc_profile_begin(), "crc_profile_begin")


def crc_profile_end() -> dict:
    kt = crc_kernel_times()
    _ck(load().crc_profile_end(ctypes.byref(kt)), "crc_profile_end")
    return {k: {"launches": int(kt.launches[i]), "ms": float(kt.ms[i])}
            for k, i in KERNEL_KINDS.items()}


def crc_synth_hidden(B, T, L, d, t0, seed, rho_t, rho_l, attempts_ptr, hidden_ptr, carry_ptr,
                     stream=None):
    _ck(load().crc_synth_hidden(B, T, L, d, t0, seed, rho_t, rho_l, attempts_ptr, hidden_ptr,
                                carry_ptr, _stream(stream)), "crc_synth_hidden")


def crc_synth_weights(L, N, d, seed, copy_init, w_ptr, stream=None):
    _ck(load().crc_synth_weights(L, N, d, seed, int(copy_init), w_ptr, _stream(stream)),
        "crc_synth_weights")


# --------------------------------------------------------------------------- #
# torch conveniences (allocation and marshalling only)
# --------------------------------------------------------------------------- #
def problem(L, N, K, d, C, R, B, expert_bytes) -> crc_problem:
    return crc_problem(L=L, N=N, K=K, d=d, C=C, R=R, B=B, reserved=0,
                       expert_bytes=int(expert_bytes))


def problem_of(w) -> crc_problem:
    """crc_problem from an object with fields L, N, K, d, C, R, B, expert_bytes."""
    return problem(w.L, w.N, w.K, w.d, w.C, w.R, w.B, w.expert_bytes)


class State:
    """A cache state in device memory (torch-allocated, 256-byte aligned)."""

    def __init__(self, p: crc_problem, device="cuda", stream=None):
        import torch
        self.p = p
        self.nbytes = crc_state_bytes(p)
        if self.nbytes == 0:
            raise CrcError(CRC_EINVAL, "crc_state_bytes")
        self.buf = torch.empty(self.nbytes, dtype=torch.uint8, device=device)
        assert self.buf.data_ptr() % 256 == 0
        self.init(stream)

    @property
    def ptr(self) -> int:
        return self.buf.data_ptr()

    def init(self, stream=None):
        crc_state_init(self.p, self.ptr, self.nbytes, stream)

    def read(self, stream=None, **kw) -> dict:
        return crc_state_read(self.p, self.ptr, self.nbytes, stream, **kw)

    def read_aux(self, stream=None) -> np.ndarray:
        return crc_state_read_aux(self.p, self.ptr, self.nbytes, stream)


@dataclass
class Trace:
    topk: object
    misses: object
    proactive: object
    cache_mid: object = None
    cache_after: object = None
    topk_set: object = None

    @staticmethod
    def alloc(p: crc_problem, T: int, device="cuda", caches: bool = False,
              rank_order: bool = True, topk_set: bool = False) -> "Trace":
        """caches: also the cache sets after the refinement and after the update
        ([B][T][L][NW] uint32 bitmasks); rank_order=False leaves out the Top-K
        in rank order (such a trace keeps crc_route_and_cache on its fused
        kernel); topk_set: the Top-K as a [B][T][L][NW] bitmask."""
        import torch
        nw = (p.N + 31) // 32

        def words(on):
            return torch.zeros((p.B, T, p.L, nw), dtype=torch.int32, device=device) if on else None

        return Trace(torch.zeros((p.B, T, p.L, p.K), dtype=torch.uint8, device=device)
                     if rank_order else None,
                     torch.zeros((p.B, T, p.L), dtype=torch.uint8, device=device),
                     torch.zeros((p.B, T, p.L), dtype=torch.uint8, device=device),
                     words(caches), words(caches), words(topk_set))

    def c(self) -> crc_trace:
        return crc_trace(_ptr(self.topk), _ptr(self.misses), _ptr(self.proactive),
                         _ptr(self.cache_mid), _ptr(self.cache_after), _ptr(self.topk_set))


def transfer_plan(p: crc_problem, cache_mid, cache_after, slot_expert=None, start=None):
    """crc_transfer_plan for one stream: cache_mid / cache_after [T][L][NW]
    (host arrays, uint32 bit patterns).  Returns (plan, slot_expert after the
    last token); plan is a structured array of TRANSFER_DTYPE."""
    mid = np.ascontiguousarray(cache_mid).view(np.uint32)
    aft = np.ascontiguousarray(cache_after).view(np.uint32)
    T = mid.shape[0]
    se = (np.full((p.L, p.C), -1, np.int32) if slot_expert is None
          else np.ascontiguousarray(slot_expert, dtype=np.int32).copy())
    st = None if start is None else np.ascontiguousarray(start).view(np.uint32)
    args = (mid.ctypes.data, aft.ctypes.data, None if st is None else st.ctypes.data)
    scratch = se.copy()                      # the counting pass moves a copy of the map
    n = crc_transfer_plan(p, T, *args, scratch.ctypes.data, None, 0)
    plan = np.zeros(n, TRANSFER_DTYPE)
    crc_transfer_plan(p, T, *args, se.ctypes.data, plan.ctypes.data if n else None, n)
    return plan, se


def transfer_replay(p: crc_problem, plan, pool, slots, pool_experts=None, stream=None):
    """crc_transfer_replay: pool a pinned host tensor of pool_experts expert
    images (default: all of it), slots a device tensor [L][C][expert_bytes]."""
    plan = np.ascontiguousarray(plan, dtype=TRANSFER_DTYPE)
    nbytes = pool.numel() * pool.element_size()
    pe = pool_experts or nbytes // int(p.expert_bytes)
    crc_transfer_replay(p, plan.ctypes.data if len(plan) else None, len(plan), pool.data_ptr(),
                        pe, slots.data_ptr(), stream)


def route_scores(p: crc_problem, hidden, w_cat, heads: int = 3, out=None, stream=None):
    import torch
    B, T, L, d = hidden.shape
    if out is None:
        out = torch.empty((B, T, L, 3, p.N), dtype=torch.float32, device=hidden.device)
    crc_route_scores(p, hidden.data_ptr(), w_cat.data_ptr(), T, heads, out.data_ptr(), stream)
    return out


def cache_scan(p: crc_problem, scores, state: State, trace: Trace | None = None, stream=None):
    T = scores.shape[1]
    crc_cache_scan(p, scores.data_ptr(), T, state.ptr, state.nbytes,
                   None if trace is None else trace.c(), stream)


def cache_scan_policy(p: crc_problem, scores, state: State, policy, trace: Trace | None = None,
                      lambda_halves: int = 1, stream=None):
    """crc_cache_scan_policy: policy is a CRC_POLICY_* value or one of POLICIES."""
    T = scores.shape[1]
    code = POLICIES[policy] if isinstance(policy, str) else int(policy)
    crc_cache_scan_policy(p, scores.data_ptr(), T, state.ptr, state.nbytes,
                          None if trace is None else trace.c(), code, lambda_halves, stream)


def cache_loss(p: crc_problem, probs, top_b: int, tau: float, w_T: float = 1.0,
               w_ST: float = 1.0, heads: int = 3, grad: bool = True, loss=None, means=None,
               grad_out=None, workspace=None, stream=None):
    """crc_cache_loss over probs [B][T][L][3][N] (fp32, on the device).

    Returns (loss [B][T][L][2] fp32, means [2] fp64 = (L_T, L_ST), grad
    [B][T][L][3][N] fp32 or None); pass preallocated tensors to reuse them."""
    import torch
    B, T, L, H, N = probs.shape
    dev = probs.device
    if loss is None:
        loss = torch.empty((B, T, L, 2), dtype=torch.float32, device=dev)
    if means is None:
        means = torch.empty(2, dtype=torch.float64, device=dev)
    if grad and grad_out is None:
        grad_out = torch.zeros((B, T, L, 3, N), dtype=torch.float32, device=dev)
    if workspace is None:
        workspace = torch.empty(max(crc_loss_workspace_bytes(p, T), 256), dtype=torch.uint8,
                                device=dev)
    crc_cache_loss(p, probs.data_ptr(), T, heads, top_b, tau, w_T, w_ST, loss.data_ptr(),
                   means.data_ptr(), grad_out.data_ptr() if grad else None, workspace.data_ptr(),
                   workspace.numel(), stream)
    return loss, means, (grad_out if grad else None)


def route_and_cache(p: crc_problem, hidden, w_cat, state: State, trace: Trace | None = None,
                    workspace=None, stream=None):
    import torch
    T = hidden.shape[1]
    if workspace is None:
        workspace = torch.empty(crc_workspace_bytes(p, T), dtype=torch.uint8,
                                device=hidden.device)
    crc_route_and_cache(p, hidden.data_ptr(), w_cat.data_ptr(), T, state.ptr, state.nbytes,
                        None if trace is None else trace.c(), workspace.data_ptr(),
                        workspace.numel() * workspace.element_size(), stream)
    return workspace


def route_and_cache_host(p: crc_problem, hidden_host, w_cat, state: State, chunk_tokens=128,
                         staging=None, workspace=None, stream=None):
    """The step on hidden states [B][T][L][d] bf16 held in (pinned) host memory:
    chunked copies overlapped with the fused step.  Returns (staging, workspace)
    for reuse; neither may be reused before `stream` has passed this call."""
    import torch
    if hidden_host.device.type != "cpu" or not hidden_host.is_contiguous():
        raise ValueError("hidden_host must be a contiguous host tensor")
    T = hidden_host.shape[1]
    dev = w_cat.device
    chunk = max(1, min(chunk_tokens, T))
    if staging is None:
        staging = torch.empty(crc_host_staging_bytes(p, chunk), dtype=torch.uint8, device=dev)
    if workspace is None:
        workspace = torch.empty(crc_fused_workspace_bytes(p), dtype=torch.uint8, device=dev)
    crc_route_and_cache_host(p, hidden_host.data_ptr(), w_cat.data_ptr(), T, chunk_tokens,
                             state.ptr, state.nbytes, staging.data_ptr(),
                             staging.numel() * staging.element_size(), workspace.data_ptr(),
                             workspace.numel() * workspace.element_size(), stream)
    return staging, workspace


def synth_weights(L, N, d, seed=0, copy_init=False, device="cuda", stream=None):
    import torch
    w = torch.empty((L, 3 * N, d), dtype=torch.bfloat16, device=device)
    crc_synth_weights(L, N, d, seed, copy_init, w.data_ptr(), stream)
    return w


def synth_hidden(B, T, L, d, seed=0, rho_t=0.9, rho_l=0.8, t0=0, carry=None, attempts=None,
                 out=None, device="cuda", stream=None):
    """Tokens [t0, t0+T) of the synthetic hidden-state field; returns (hidden, carry)."""
    import torch
    if out is None:
        out = torch.empty((B, T, L, d), dtype=torch.bfloat16, device=device)
    if carry is None:
        carry = torch.zeros((B, L, d), dtype=torch.float32, device=device)
    crc_synth_hidden(B, T, L, d, t0, seed, rho_t, rho_l, _ptr(attempts), out.data_ptr(),
                     carry.data_ptr(), stream)
    return out, carry


def _stats_struct(stats: dict) -> crc_stats:
    st = crc_stats()
    for f, _ in crc_stats._fields_:
        if f in stats and f != "reserved":
            setattr(st, f, int(stats[f]))
    return st


def load_time(stats: dict, p: crc_problem, c_exp: float, eta: float) -> float:
    """crc_load_time: exposed expert-loading cost per decode token under the
    paper's overlap model, from the totals of crc_state_read (a dict as
    returned by State.read)."""
    if not 0.0 <= eta <= 1.0:
        raise ValueError("eta must lie in [0, 1]")
    out = ctypes.c_double()
    _ck(load().crc_load_time(ctypes.byref(p), ctypes.byref(_stats_struct(stats)), c_exp, eta,
                             ctypes.byref(out)), "crc_load_time")
    return out.value


def metrics(stats: dict, p: crc_problem) -> dict:
    """crc_metrics: Hit, AdjHit, traffic and Load/token (bytes per decode
    token) of Sec. 4.1 from the totals of crc_state_read."""
    r = crc_report()
    _ck(load().crc_metrics(ctypes.byref(p), ctypes.byref(_stats_struct(stats)), ctypes.byref(r)),
        "crc_metrics")
    return {"hit": r.hit, "adj_hit": r.adj_hit, "traffic_bytes": r.traffic_bytes,
            "load_per_token_bytes": r.load_per_token_bytes}
