"""CPU oracle for cache-aware MoE routing and expert residency.

TEST INFRASTRUCTURE ONLY: imported by ``tests/``, ``__graft_entry__.smoke()``
and the CPU-baseline leg of ``bench.py``; never by the product package.

The arithmetic lives in ``crc_oracle.c`` / ``scan_body.h`` (plain C, fp64
router and softmax, literal Algorithms 1 and 2 of the paper).  This module
compiles it with gcc and wraps it with ctypes.

Parity pins (see ``tests/test_oracle_*.py``): brute force over all small
caches and score orders, the closed forms of Algorithms 1 and 2 on a full
cache, the special cases C = K (R = 0), C = N, constant hidden state, R = 0
equals update-only, copy-initialised heads, a library softmax cross-check,
the published Philox test vectors for the input generator, hand-traced
worked examples (``tests/test_oracle_scan.py``), hand-built accesses whose
closest decision is known (``tests/test_oracle_margins.py``) and the paper's
printed metric identities (Table 1, Table 2; ``tests/golden/``).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD = os.path.join(_HERE, "_build")
_SO = os.path.join(_BUILD, "libcrc_oracle.so")
_SRC = [os.path.join(_HERE, "crc_oracle.c"), os.path.join(_HERE, "scan_body.h")]
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle into oracle/_build/libcrc_oracle.so (host compiler only)."""
    os.makedirs(_BUILD, exist_ok=True)
    stale = force or not os.path.exists(_SO) or any(
        os.path.getmtime(s) > os.path.getmtime(_SO) for s in _SRC)
    if stale:
        tmp = _SO + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-pthread",
               "-ffp-contract=off", "-fno-fast-math", "-Wall", "-Wno-unused-function",
               "-o", tmp, _SRC[0], "-lm"]
        subprocess.run(cmd, check=True, cwd=_HERE)
        os.replace(tmp, _SO)
    return _SO


def lib():
    global _lib
    with _lock:
        if _lib is None:
            build()
            L = ctypes.CDLL(_SO)
            P = ctypes.c_void_p
            i = ctypes.c_int
            L.oracle_unit_probs.argtypes = [i, i, i, P, P, P]
            L.oracle_router_probs.argtypes = [i, i, i, i, i, i, P, P, P, i]
            for sfx in ("f64", "f32"):
                f = getattr(L, f"oracle_step_{sfx}")
                f.argtypes = [i, i, i, i, i, P, P, P, P, P, P, P, P, P, P]
                f.restype = i
                f = getattr(L, f"oracle_scan_{sfx}")
                f.argtypes = [i, i, i, i, i, i, i, P, P, P, P, P, P, P, P, i, i]
                f.restype = i
                f = getattr(L, f"oracle_refine_{sfx}")
                f.argtypes = [i, i, i, P, P, P, P]
                f.restype = i
                f = getattr(L, f"oracle_update_cache_{sfx}")
                f.argtypes = [i, i, P, P, P, P, P]
                f.restype = i
            d = ctypes.c_double
            L.oracle_metrics.argtypes = [d, d, d, d, d, P, P, P]
            _lib = L
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def default_threads() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:  # pragma: no cover
        return os.cpu_count() or 1


# --------------------------------------------------------------------------- #
def unit_probs(h_row_bits: np.ndarray, w_layer_bits: np.ndarray, N: int, H: int = 3) -> np.ndarray:
    """fp64 [H][N] probabilities of one unit (Sec. 2, 3.2, 3.3)."""
    h = np.ascontiguousarray(h_row_bits, dtype=np.uint16)
    w = np.ascontiguousarray(w_layer_bits, dtype=np.uint16)
    d = h.shape[-1]
    assert w.shape[-1] == d and w.shape[0] >= H * N
    out = np.zeros((H, N), dtype=np.float64)
    lib().oracle_unit_probs(N, d, H, _ptr(h), _ptr(w), _ptr(out))
    return out


def router_probs(hidden_bits: np.ndarray, w_bits: np.ndarray, N: int, H: int = 3,
                 nthreads: int | None = None) -> np.ndarray:
    """fp64 probabilities [B][T][L][3][N] from bf16 bits hidden [B][T][L][d], W [L][3N][d]."""
    h = np.ascontiguousarray(hidden_bits, dtype=np.uint16)
    w = np.ascontiguousarray(w_bits, dtype=np.uint16)
    B, T, L, d = h.shape
    assert w.shape == (L, 3 * N, d), (w.shape, (L, 3 * N, d))
    out = np.zeros((B, T, L, 3, N), dtype=np.float64)
    lib().oracle_router_probs(B, T, L, N, d, H, _ptr(h), _ptr(w), _ptr(out),
                              nthreads or default_threads())
    return out


def scan(probs: np.ndarray, K: int, C: int, R: int, trace: bool = True,
         margins: bool = False, nthreads: int | None = None,
         exact_ties_exempt: bool = False) -> dict:
    """Literal Algorithm 2 + 1 over [B][T][L][3][N] probabilities.

    fp64 input runs the fp64 scan; fp32 input runs the fp32 scan (every sum
    and comparison in fp32).  Returns the trace, the final caches and the
    per-(stream, layer) counters (hits, demand misses, proactive loads).
    margins: each access's decision margin, the smallest relative gap between
    the two scores of any decision it took; exact_ties_exempt leaves gaps of
    exactly zero out of it (ties built on purpose, broken by index on every
    side).
    """
    if probs.dtype == np.float64:
        sfx = "f64"
    elif probs.dtype == np.float32:
        sfx = "f32"
    else:
        raise TypeError(probs.dtype)
    p = np.ascontiguousarray(probs)
    B, T, L, three, N = p.shape
    assert three == 3
    NW = (N + 31) // 32
    res = {
        "topk": np.zeros((B, T, L, K), np.uint8) if trace else None,
        "misses": np.zeros((B, T, L), np.uint8) if trace else None,
        "proactive": np.zeros((B, T, L), np.uint8) if trace else None,
        "margins": np.zeros((B, T, L), np.float64) if margins else None,
        "cache_bits": np.zeros((B, L, NW), np.uint32),
        "aT": np.zeros((B, L, N), p.dtype),
        "counters": np.zeros((B, L, 3), np.uint64),
    }
    rc = getattr(lib(), f"oracle_scan_{sfx}")(
        B, T, L, N, K, C, R, _ptr(p), _ptr(res["topk"]), _ptr(res["misses"]),
        _ptr(res["proactive"]), _ptr(res["margins"]), _ptr(res["cache_bits"]),
        _ptr(res["aT"]), _ptr(res["counters"]), nthreads or default_threads(),
        int(exact_ties_exempt))
    if rc != 0:
        raise ValueError("oracle_scan rejected the sizes")
    return res


# comparison policies (numbering shared with nothing: the oracle's own)
POLICIES = {"lru": 1, "lfu": 2, "lrfu": 3, "spatio_lru": 4}


def policy_scan(probs: np.ndarray, K: int, C: int, R: int, policy: str, lambda2: int = 1,
                trace: bool = True) -> dict:
    """Cache scan under a comparison policy (LRU, LFU, LRFU with
    lambda = lambda2 / 2, Spatio-only with LRU demand eviction) over fp32
    probabilities [B][T][L][3][N]; see the readings in crc_oracle.c."""
    p = np.ascontiguousarray(probs, dtype=np.float32)
    B, T, L, three, N = p.shape
    assert three == 3
    NW = (N + 31) // 32
    res = {
        "topk": np.zeros((B, T, L, K), np.uint8) if trace else None,
        "misses": np.zeros((B, T, L), np.uint8) if trace else None,
        "proactive": np.zeros((B, T, L), np.uint8) if trace else None,
        "cache_bits": np.zeros((B, L, NW), np.uint32),
        "aux": np.zeros((B, L, N), np.uint32),
        "val": np.zeros((B, L, N), np.float32),
        "counters": np.zeros((B, L, 3), np.uint64),
    }
    rc = lib().oracle_policy_scan(B, T, L, N, K, C, R, POLICIES[policy], lambda2, _ptr(p),
                                  _ptr(res["topk"]), _ptr(res["misses"]), _ptr(res["proactive"]),
                                  _ptr(res["cache_bits"]), _ptr(res["aux"]), _ptr(res["val"]),
                                  _ptr(res["counters"]))
    if rc != 0:
        raise ValueError("oracle_policy_scan rejected the sizes")
    return res


def cache_loss(probs: np.ndarray, top_b: int, tau: float, w_T: float = 1.0, w_ST: float = 1.0,
               grad: bool = True, grad_p: bool = False) -> dict:
    """Soft Top-B coverage losses (Sec. 3.1-3.3) over fp32 probabilities
    [B][T][L][3][N]: per-unit l^T and l^ST [B][T][L][2], their means over the
    valid positions, and the gradient of w_T L_T + w_ST L_ST with respect to
    the three heads' logits [B][T][L][3][N] (fp64); the native distributions
    are differentiable both as priorities and as targets (Sec. 3.4).
    grad_p adds the gradient with respect to the probabilities ("grad_p")."""
    p = np.ascontiguousarray(probs, dtype=np.float32)
    B, T, L, three, N = p.shape
    assert three == 3
    loss = np.zeros((B, T, L, 2), np.float32)
    g = np.zeros(p.shape, np.float64) if grad else None
    gp = np.zeros(p.shape, np.float64) if grad_p else None
    rc = lib().oracle_cache_loss(B, T, L, N, top_b, ctypes.c_double(tau), ctypes.c_double(w_T),
                                 ctypes.c_double(w_ST), _ptr(p), _ptr(loss), _ptr(g), _ptr(gp))
    if rc != 0:
        raise ValueError("oracle_cache_loss rejected the sizes")
    n = B * (T - 1) * L
    return {"loss": loss, "grad": g, "grad_p": gp,
            "L_T": float(loss[..., 0].astype(np.float64).sum() / n) if n else 0.0,
            "L_ST": float(loss[..., 1].astype(np.float64).sum() / n) if n else 0.0}


class Chain:
    """State of one (stream, layer) chain for step-by-step replay."""

    def __init__(self, N: int, dtype=np.float64):
        self.N = N
        self.dtype = np.dtype(dtype)
        self.in_cache = np.zeros(N, np.uint8)
        self.count = ctypes.c_int(0)
        self.aT = np.zeros(N, self.dtype)

    def copy(self) -> "Chain":
        c = Chain(self.N, self.dtype)
        c.in_cache[:] = self.in_cache
        c.count.value = self.count.value
        c.aT[:] = self.aT
        return c

    def members(self) -> set:
        return {int(e) for e in np.flatnonzero(self.in_cache)}


def step(chain: Chain, t: int, K: int, C: int, R: int, pR, pT, pS_pred=None):
    """One access (Algorithm 2 then Algorithm 1).  Returns (topk, misses, proactive, margin)."""
    dt = chain.dtype
    sfx = "f64" if dt == np.float64 else "f32"
    pR = np.ascontiguousarray(pR, dtype=dt)
    pT = np.ascontiguousarray(pT, dtype=dt)
    pS = None if pS_pred is None else np.ascontiguousarray(pS_pred, dtype=dt)
    if R > 0 and t >= 1 and pS is None:
        raise ValueError("refinement needs p^S of the causal predecessor")
    topk = np.zeros(K, np.int32)
    mi, pr, mg = ctypes.c_int(0), ctypes.c_int(0), ctypes.c_double(0)
    rc = getattr(lib(), f"oracle_step_{sfx}")(
        chain.N, K, C, R, t, _ptr(pR), _ptr(pT), _ptr(pS), _ptr(chain.in_cache),
        ctypes.byref(chain.count), _ptr(chain.aT), _ptr(topk), ctypes.byref(mi),
        ctypes.byref(pr), ctypes.byref(mg))
    if rc != 0:
        raise ValueError("oracle_step rejected the sizes")
    return [int(x) for x in topk], mi.value, pr.value, mg.value


def metrics(A: float, D: float, P: float, T: float, s_exp_bytes: float) -> dict:
    """Hit, AdjHit and Load/token (bytes per token) as defined in Sec. 4.1."""
    h, a, ld = ctypes.c_double(), ctypes.c_double(), ctypes.c_double()
    lib().oracle_metrics(float(A), float(D), float(P), float(T), float(s_exp_bytes),
                         ctypes.byref(h), ctypes.byref(a), ctypes.byref(ld))
    return {"hit": h.value, "adj_hit": a.value, "load_per_token": ld.value}


def load_time(D: float, P: float, T: float, c_exp: float, eta: float) -> float:
    """Modeled exposed expert-loading cost per decode token (appendix on
    asynchronous transfer overlap): c_exp / T * (D + (1 - eta) * P)."""
    f = lib().oracle_load_time
    f.restype = ctypes.c_double
    f.argtypes = [ctypes.c_double] * 5
    return f(float(D), float(P), float(T), float(c_exp), float(eta))


def run(hidden_bits: np.ndarray, w_bits: np.ndarray, N: int, K: int, C: int, R: int,
        margins: bool = True, nthreads: int | None = None,
        exact_ties_exempt: bool = False) -> dict:
    """End-to-end fp64 oracle: router probabilities then the scan."""
    H = 3 if R > 0 else 2
    p = router_probs(hidden_bits, w_bits, N, H, nthreads)
    res = scan(p, K, C, R, trace=True, margins=margins, nthreads=nthreads,
               exact_ties_exempt=exact_ties_exempt)
    res["probs"] = p
    return res


def bits_to_sets(cache_bits: np.ndarray, N: int):
    """[..., NW] uint32 bitmasks -> nested lists of expert sets."""
    flat = cache_bits.reshape(-1, cache_bits.shape[-1])
    out = []
    for row in flat:
        out.append({e for e in range(N) if (int(row[e // 32]) >> (e % 32)) & 1})
    return np.array(out, dtype=object).reshape(cache_bits.shape[:-1])


def refine(in_cache: np.ndarray, sST, C: int, R: int, dtype=np.float64):
    """Algorithm 2's refinement loop on a copy of in_cache.  Returns (new_in_cache, proactive, margin)."""
    dt = np.dtype(dtype)
    sfx = "f64" if dt == np.float64 else "f32"
    ic = np.array(in_cache, dtype=np.uint8)
    s = np.ascontiguousarray(sST, dtype=dt)
    cnt = ctypes.c_int(int(ic.sum()))
    mg = ctypes.c_double(float("inf"))
    p = getattr(lib(), f"oracle_refine_{sfx}")(len(ic), C, R, _ptr(s), _ptr(ic),
                                               ctypes.byref(cnt), ctypes.byref(mg))
    return ic, p, mg.value


def update_cache(in_cache: np.ndarray, S, s, C: int, dtype=np.float64):
    """Algorithm 1 on a copy of in_cache.  Returns (new_in_cache, |D|, margin)."""
    dt = np.dtype(dtype)
    sfx = "f64" if dt == np.float64 else "f32"
    ic = np.array(in_cache, dtype=np.uint8)
    inS = np.zeros(len(ic), np.uint8)
    inS[list(S)] = 1
    sv = np.ascontiguousarray(s, dtype=dt)
    cnt = ctypes.c_int(int(ic.sum()))
    mg = ctypes.c_double(float("inf"))
    nd = getattr(lib(), f"oracle_update_cache_{sfx}")(len(ic), C, _ptr(sv), _ptr(inS), _ptr(ic),
                                                     ctypes.byref(cnt), ctypes.byref(mg))
    return ic, nd, mg.value
