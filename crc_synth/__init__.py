"""Seeded synthetic inputs for the cache-aware routing path (numpy, host side).

This module holds no arithmetic of the method itself (no router, softmax,
Top-K or cache policy).  It only draws the inputs both sides consume:

* hidden states ``h[b, t, l, :]`` in bf16, laid out ``[B][T][L][d]``;
* router weights ``W_cat[l, head*N + e, :]`` in bf16, laid out ``[L][3N][d]``,
  heads ordered native (R), Temporal (T), Spatio (S).

Generator definition (the CUDA generator in the library implements the same
definition independently and must reproduce these bits exactly):

1. Counter-based uniform bits: Philox4x32-10 (Salmon, Moraes, Dror, Shaw,
   "Parallel Random Numbers: As Easy as 1, 2, 3", SC'11), key
   ``(seed, tag)``, 10 rounds, multipliers 0xD2511F53 / 0xCD9E8D57 and key
   increments 0x9E3779B9 / 0xBB67AE85.
2. One Philox call yields four 32-bit words = eight 16-bit integers
   ``u0..u7`` (low half of each word first).  Two variates come out of one
   call: ``eps_even`` from ``u0..u3`` and ``eps_odd`` from ``u4..u7`` by the
   Irwin-Hall sum of four uniforms, centred and scaled to unit variance,
   all in fp32: ``fp32(u0+u1+u2+u3 - 131070) * c`` with
   ``c = fp32(sqrt(3 / (65536**2 - 1)))`` (bits 0x37ddb3d7).  The sum is an
   exact integer and the single multiply is correctly rounded, so the value
   is the same on every IEEE machine.
3. Hidden states follow a separable AR(1) field, unit variance, correlation
   ``rho_t**|dt| * rho_l**|dl|``: first an AR(1) over layers driven by the
   innovations, ``g[t,0] = eps[t,0]``, ``g[t,l] = rho_l*g[t,l-1] + s_l*eps[t,l]``,
   then an AR(1) over tokens driven by ``g``: ``h[0,l] = g[0,l]``,
   ``h[t,l] = rho_t*h[t-1,l] + s_t*g[t,l]``, with ``s = fp32(sqrt(1-rho^2))``.
   Each product and sum is a separate fp32 operation (no fused multiply-add),
   evaluated in exactly that order.  The stored value is ``bf16_rne(h)``.
   Innovation counters: ``(j, l, t, b | attempt << 16)`` with ``j = i // 2``
   (element ``i`` takes ``eps_even`` when even, ``eps_odd`` when odd), key
   ``(seed, TAG_HIDDEN)``.  ``attempt`` (0 unless a re-draw table is given)
   lets a test re-draw the innovations of one unit without touching others.
4. Weights: ``W[l, h*N+e, i] = bf16_rne(eps * fp32(1/sqrt(d)))`` (i.e. N(0, 1/d)),
   counters ``(j, e, h, l)``, key ``(seed, TAG_WEIGHT)``.  ``copy_init``
   replaces the Temporal and Spatio heads by copies of native rows following
   the paper's router initialisation (Sec. 3.4): ``W^T_l = W^R_l``,
   ``W^S_l = W^R_{l+1}``, ``W^S_L = W^R_1``.

The workload shapes mirror the backbones the paper evaluates (Sec. 4.1:
Qwen3-30B-A3B with L=48, N=128, K=8; GPT-OSS-20B with L=24, N=32, K=4) and
stand in for its decoding traces on GSM8K / MATH / CommonsenseQA, which are
not available here.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

TAG_HIDDEN = 0x48494444   # "HIDD"
TAG_WEIGHT = 0x57474854   # "WGHT"

_M0 = np.uint64(0xD2511F53)
_M1 = np.uint64(0xCD9E8D57)
_W0 = 0x9E3779B9
_W1 = 0xBB67AE85
_MASK32 = np.uint64(0xFFFFFFFF)
_IH_SCALE = np.uint32(0x37DDB3D7).view(np.float32)   # fp32(sqrt(3/(65536^2-1)))


# --------------------------------------------------------------------------- #
# Problem shapes
# --------------------------------------------------------------------------- #
@dataclass(frozen=True)
class Workload:
    """One synthetic workload: the problem statement's sizes plus generator knobs."""
    name: str
    L: int
    N: int
    K: int
    d: int
    C: int
    R: int
    B: int
    T: int
    expert_bytes: int
    rho_t: float = 0.9
    rho_l: float = 0.8
    extra: dict = field(default_factory=dict, compare=False)

    @property
    def units(self) -> int:
        return self.B * self.T * self.L

    def with_(self, **kw) -> "Workload":
        d = dict(self.__dict__)
        d.update(kw)
        return Workload(**d)


# The five configurations: a tiny one, two backbone-shaped ones, the
# update-only capacity sweep and a large streamed one.
TINY = Workload("tiny", L=4, N=16, K=2, d=256, C=4, R=1, B=4, T=256,
                expert_bytes=1 << 20)
QWEN3_30B = Workload("qwen3-30b-a3b", L=48, N=128, K=8, d=2048, C=32, R=4, B=64,
                     T=1024, expert_bytes=3 * 2048 * 768 * 2)
GPT_OSS_20B = Workload("gpt-oss-20b", L=24, N=32, K=4, d=2880, C=8, R=2, B=128,
                       T=2048, expert_bytes=3 * 2880 * 2880 * 2, rho_t=0.85)
SWEEP_R0 = Workload("qwen3-30b-sweep-r0", L=48, N=128, K=8, d=2048, C=32, R=0,
                    B=256, T=2048, expert_bytes=3 * 2048 * 768 * 2,
                    extra={"C_values": (16, 32, 64, 96)})
# Expert size for the 235B shape is not given; 3*4096*1536*2 is the
# Qwen3-235B-A22B expert (gate, up, down at d=4096, moe_ffn=1536) in bf16.
LARGE = Workload("qwen3-235b-a22b", L=94, N=128, K=8, d=4096, C=32, R=2, B=512,
                 T=4096, expert_bytes=3 * 4096 * 1536 * 2,
                 extra={"R_values": (2, 8), "expert_bytes_assumed": True})

WORKLOADS = {w.name: w for w in (TINY, QWEN3_30B, GPT_OSS_20B, SWEEP_R0, LARGE)}


# --------------------------------------------------------------------------- #
# Philox4x32-10 and the Irwin-Hall normal
# --------------------------------------------------------------------------- #
def philox4x32_10(c0, c1, c2, c3, k0, k1):
    """Philox4x32 with 10 rounds on broadcastable uint32 arrays.

    Returns four uint32 arrays.  Follows the published round function: the
    two multiplies take words 0 and 2, the outputs are
    ``(hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0)`` and the key is bumped by the
    Weyl constants between rounds.
    """
    c0, c1, c2, c3 = (np.asarray(x, dtype=np.uint64) for x in (c0, c1, c2, c3))
    k0 = int(k0) & 0xFFFFFFFF
    k1 = int(k1) & 0xFFFFFFFF
    for r in range(10):
        if r:
            k0 = (k0 + _W0) & 0xFFFFFFFF
            k1 = (k1 + _W1) & 0xFFFFFFFF
        p0 = _M0 * c0
        p1 = _M1 * c2
        hi0, lo0 = p0 >> np.uint64(32), p0 & _MASK32
        hi1, lo1 = p1 >> np.uint64(32), p1 & _MASK32
        c0, c1, c2, c3 = (hi1 ^ c1 ^ np.uint64(k0), lo1,
                          hi0 ^ c3 ^ np.uint64(k1), lo0)
    return tuple(x.astype(np.uint32) for x in (c0, c1, c2, c3))


def _irwin_hall4(wa, wb):
    """fp32 unit-variance variate from the four 16-bit halves of two words."""
    s = ((wa & 0xFFFF).astype(np.int64) + (wa >> 16).astype(np.int64)
         + (wb & 0xFFFF).astype(np.int64) + (wb >> 16).astype(np.int64))
    return (s - 131070).astype(np.float32) * _IH_SCALE


def normal_pairs(c0, c1, c2, c3, k0, k1):
    """Two fp32 variates (even, odd) per counter."""
    w0, w1, w2, w3 = philox4x32_10(c0, c1, c2, c3, k0, k1)
    return _irwin_hall4(w0, w1), _irwin_hall4(w2, w3)


def bf16_rne_bits(x: np.ndarray) -> np.ndarray:
    """Round fp32 to bf16 (round to nearest even); returns uint16 bit patterns."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    r = (u + np.uint64(0x7FFF) + ((u >> np.uint64(16)) & np.uint64(1))) >> np.uint64(16)
    return r.astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def ar_constants(rho: float):
    """(rho, sqrt(1-rho^2)) as fp32, computed from the double value of rho."""
    return np.float32(rho), np.float32(math.sqrt(1.0 - float(rho) * float(rho)))


# --------------------------------------------------------------------------- #
# Hidden states
# --------------------------------------------------------------------------- #
def _innovations(seed, b, t_idx, L, d, attempt=None):
    """eps[len(t_idx), L, d] fp32 for stream b.  attempt: uint8 [len(t_idx), L] or None."""
    j = np.arange(d // 2, dtype=np.uint32)
    l = np.arange(L, dtype=np.uint32)
    t = np.asarray(t_idx, dtype=np.uint32)
    c0 = j[None, None, :]
    c1 = l[None, :, None]
    c2 = t[:, None, None]
    if attempt is None:
        c3 = np.uint32(b)
    else:
        c3 = (np.uint32(b) | (attempt.astype(np.uint32) << np.uint32(16)))[:, :, None]
    c0, c1, c2, c3 = np.broadcast_arrays(c0, c1, c2, c3)
    ev, od = normal_pairs(c0, c1, c2, c3, seed, TAG_HIDDEN)
    eps = np.empty((len(t), L, d), dtype=np.float32)
    eps[..., 0::2] = ev
    eps[..., 1::2] = od
    return eps


def hidden_stream(seed: int, b: int, T: int, L: int, d: int, rho_t: float, rho_l: float,
                  attempts: np.ndarray | None = None, t_chunk: int = 256) -> np.ndarray:
    """bf16 bits [T][L][d] of stream b (see the module docstring for the definition)."""
    if d % 2:
        raise ValueError("d must be even")
    rt, st = ar_constants(rho_t)
    rl, sl = ar_constants(rho_l)
    out = np.empty((T, L, d), dtype=np.uint16)
    h_prev = None
    for t0 in range(0, T, t_chunk):
        tt = np.arange(t0, min(T, t0 + t_chunk))
        att = None if attempts is None else attempts[tt]
        eps = _innovations(seed, b, tt, L, d, att)
        g = np.empty_like(eps)
        g[:, 0] = eps[:, 0]
        for l in range(1, L):
            g[:, l] = (rl * g[:, l - 1]) + (sl * eps[:, l])
        h = np.empty_like(g)
        for k in range(len(tt)):
            if h_prev is None:
                h[k] = g[k]
            else:
                h[k] = (rt * h_prev) + (st * g[k])
            h_prev = h[k]
        out[tt] = bf16_rne_bits(h)
    return out


class HiddenWalk:
    """One stream's hidden states drawn unit by unit in causal order
    (t = 0, 1, ...; l = 0 .. L-1 within a token), with the definition of
    ``hidden_stream``: ``draw(t, l, attempt)`` proposes h[t, l] from the
    innovation of that attempt without changing the walk, ``accept`` keeps
    the proposal.  A test that redraws a unit's innovation (to move a draw
    away from an unwanted event) walks the same field ``hidden_stream``
    produces when given the accepted attempts as its re-draw table."""

    def __init__(self, seed: int, b: int, L: int, d: int, rho_t: float, rho_l: float):
        if d % 2:
            raise ValueError("d must be even")
        self.seed, self.b, self.L, self.d = seed, b, L, d
        self.rt, self.st = ar_constants(rho_t)
        self.rl, self.sl = ar_constants(rho_l)
        self.h_prev = None            # h[t-1, :] fp32 [L][d]
        self.h_cur = np.empty((L, d), np.float32)
        self.g_prev = None            # g[t, l-1] fp32 [d]
        self._t = -1
        self._eps0 = None             # innovations of attempt 0 for token t, [L][d]

    def _eps(self, t: int, l: int, attempt: int) -> np.ndarray:
        if attempt == 0:
            if self._t != t:
                self._eps0 = _innovations(self.seed, self.b, [t], self.L, self.d)[0]
                self._t = t
            return self._eps0[l]
        j = np.arange(self.d // 2, dtype=np.uint32)
        c3 = np.uint32(self.b) | (np.uint32(attempt) << np.uint32(16))
        ev, od = normal_pairs(j, np.uint32(l), np.uint32(t), c3, self.seed, TAG_HIDDEN)
        e = np.empty(self.d, np.float32)
        e[0::2] = ev
        e[1::2] = od
        return e

    def draw(self, t: int, l: int, attempt: int = 0):
        """Proposal for unit (t, l): (bf16 bits [d], state to pass to accept)."""
        eps = self._eps(t, l, attempt)
        g = eps.copy() if l == 0 else (self.rl * self.g_prev) + (self.sl * eps)
        h = g.copy() if self.h_prev is None else (self.rt * self.h_prev[l]) + (self.st * g)
        return bf16_rne_bits(h), (t, l, g, h)

    def accept(self, state) -> None:
        t, l, g, h = state
        self.g_prev = g
        self.h_cur[l] = h
        if l == self.L - 1:
            self.h_prev = self.h_cur.copy()


def hidden(w: Workload, seed: int = 0, streams=None, T: int | None = None,
           attempts: np.ndarray | None = None) -> np.ndarray:
    """bf16 bits [len(streams)][T][L][d] (all streams by default)."""
    T = w.T if T is None else T
    streams = range(w.B) if streams is None else streams
    return np.stack([hidden_stream(seed, b, T, w.L, w.d, w.rho_t, w.rho_l,
                                   None if attempts is None else attempts[b])
                     for b in streams])


# --------------------------------------------------------------------------- #
# Router weights
# --------------------------------------------------------------------------- #
def weights(w: Workload, seed: int = 0, copy_init: bool = False) -> np.ndarray:
    """bf16 bits [L][3N][d]: heads R, T, S, each N(0, 1/d)."""
    L, N, d = w.L, w.N, w.d
    scale = np.float32(1.0 / math.sqrt(d))
    out = np.empty((L, 3 * N, d), dtype=np.uint16)
    j = np.arange(d // 2, dtype=np.uint32)[None, :]
    e = np.arange(N, dtype=np.uint32)[:, None]
    for l in range(L):
        for h in range(3):
            c0, c1 = np.broadcast_arrays(j, e)
            ev, od = normal_pairs(c0, c1, np.uint32(h), np.uint32(l), seed, TAG_WEIGHT)
            x = np.empty((N, d), dtype=np.float32)
            x[:, 0::2] = ev * scale
            x[:, 1::2] = od * scale
            out[l, h * N:(h + 1) * N] = bf16_rne_bits(x)
    if copy_init:
        for l in range(L):
            out[l, N:2 * N] = out[l, 0:N]
            out[l, 2 * N:3 * N] = out[(l + 1) % L, 0:N]
    return out


def near_uniform_scores(shape, seed: int, lo: float = 1e-6) -> np.ndarray:
    """Positive fp32 values in [lo, 1) from Philox, for exercising the scan alone."""
    n = int(np.prod(shape))
    half = (n + 1) // 2
    idx = np.arange(half, dtype=np.uint32)
    w0, w1, w2, w3 = philox4x32_10(idx, np.uint32(0), np.uint32(0), np.uint32(0), seed, 0x53434F52)
    u = np.empty(2 * half, dtype=np.float64)
    u[0::2] = (w0 >> 8).astype(np.float64) / 16777216.0
    u[1::2] = (w2 >> 8).astype(np.float64) / 16777216.0
    return np.maximum(u[:n], lo).astype(np.float32).reshape(shape)


def distributions(B: int, T: int, L: int, N: int, seed: int, rho: float = 0.6,
                  power: float = 20.0, quant: int | None = None, streams=None) -> np.ndarray:
    """Router-like probability rows fp32 [B][T][L][3][N] for exercising the
    coverage losses alone (host PCG64, one generator per stream).

    Each row is a normalised positive draw: x_t = rho x_{t-1} + (1 - rho) u_t^power
    with u ~ U(0, 1) per (stream, token, layer, head, expert), so a few experts
    dominate each row and neighbouring tokens stay similar, then p = x / sum x.
    quant rounds to multiples of 1/quant afterwards (ties on purpose).  streams
    selects a subset of the B streams (the same rows as in the full draw).
    With the defaults at N = 128 the top 8 experts hold about 0.36 of a row's
    mass and consecutive tokens correlate at about 0.6."""
    idx = range(B) if streams is None else streams
    out = np.empty((len(idx), T, L, 3, N), np.float32)
    for i, b in enumerate(idx):
        rng = np.random.default_rng([seed, b])
        u = rng.random((T, L, 3, N), dtype=np.float32) ** np.float32(power)
        x = np.empty_like(u)
        x[0] = u[0]
        for t in range(1, T):
            x[t] = np.float32(rho) * x[t - 1] + np.float32(1.0 - rho) * u[t]
        x += np.float32(1e-6)
        x /= x.sum(-1, keepdims=True)
        if quant:
            x = np.round(x * quant) / np.float32(quant)
        out[i] = x
    return out
