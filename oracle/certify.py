"""Margin-certified inputs for end-to-end parity against the fp64 oracle.

TEST INFRASTRUCTURE ONLY (like the rest of ``oracle/``).

The GPU decides in fp32 and the oracle in fp64, so their decisions can only
be compared where every decision the literal algorithm takes has a relative
gap of at least ``tol`` between the two scores it compares (the decision
margin of ``oracle.step``/``oracle.refine``).  This module draws a stream's
hidden states unit by unit in causal order with the generator's own walk
(``crc_synth.HiddenWalk``), runs the oracle on each unit and, when a draw
would put a decision closer than ``tol``, redraws that unit's innovation
(the generator's ``attempt`` counter, at most ``max_tries`` times).  The
decisions that depend on the draw of unit v = (t, l) are those of its own
access (the native Top-K of Sec. 2 and Algorithm 1's evictions) and the
pre-access refinement of the next unit in causal order, whose causal
predecessor v is (Sec. 3.3: rho(t, l+1) = (t, l), rho(t+1, 0) = (t, L-1));
the refinement's other inputs (the cache after the previous token and a^T)
are fixed by then.  Both are checked before a draw is kept.

The result is the accepted re-draw table (the generator reproduces the same
field from it, on the host or on the device), the hidden states, and the
fp64 oracle's per-access trace, margins and final state of each stream.
Units that no redraw could certify stay flagged (``certified`` False).
"""
from __future__ import annotations

import multiprocessing
from concurrent.futures import ProcessPoolExecutor

import numpy as np

import crc_synth as S

from . import Chain, default_threads, refine, step, unit_probs


def _certify_stream(w, W, seed: int, b: int, tol: float, max_tries: int) -> dict:
    L, N, K, C, R, T, d = w.L, w.N, w.K, w.C, w.R, w.T, w.d
    H = 3 if R > 0 else 2
    NW = (N + 31) // 32
    walk = S.HiddenWalk(seed, b, L, d, w.rho_t, w.rho_l)
    chains = [Chain(N) for _ in range(L)]
    out = {
        "attempts": np.zeros((T, L), np.uint8),
        "hidden": np.empty((T, L, d), np.uint16),
        "topk": np.zeros((T, L, K), np.uint8),
        "misses": np.zeros((T, L), np.uint8),
        "proactive": np.zeros((T, L), np.uint8),
        "margins": np.full((T, L), np.inf),
        "certified": np.zeros((T, L), bool),
        "counters": np.zeros((L, 3), np.uint64),
        "redraws": 0,
    }
    pS_prev = None          # p^S of the previous unit (the next unit's causal predecessor)
    ref_margin = np.inf     # refinement margin of the current unit, fixed by its predecessor
    for t in range(T):
        for l in range(L):
            # Algorithm 2's refinement of (t, l): its inputs are already fixed
            ch = chains[l].copy()
            pro = 0
            if R > 0 and t >= 1:
                sST = ch.aT + pS_prev
                ic, pro, m_ref = refine(ch.in_cache, sST, C, R)
                ch.in_cache[:] = ic
                ch.count.value = int(ic.sum())
                assert m_ref == ref_margin
            # the next unit in causal order, whose refinement this draw decides
            tn, ln = (t, l + 1) if l + 1 < L else (t + 1, 0)
            next_refines = R > 0 and 1 <= tn < T
            best = None
            for a in range(max_tries):
                bits, st = walk.draw(t, l, a)
                p = unit_probs(bits, W[l], N, H)
                acc = ch.copy()
                tk, mi, _, m_acc = step(acc, t, K, C, 0, p[0], p[1])   # access + UpdateCache
                m_next = np.inf
                if next_refines:
                    nxt = acc if ln == l else chains[ln]               # L = 1: this chain
                    _, _, m_next = refine(nxt.in_cache, nxt.aT + p[2], C, R)
                score = min(m_acc, m_next)
                if best is None or score > best[0]:
                    best = (score, a, bits, st, p, acc, tk, mi, m_acc, m_next)
                if score >= tol:
                    break
            score, a, bits, st, p, acc, tk, mi, m_acc, m_next = best
            out["redraws"] += a
            walk.accept(st)
            chains[l] = acc
            pS_prev = p[2] if H == 3 else None
            out["attempts"][t, l] = a
            out["hidden"][t, l] = bits
            out["topk"][t, l] = tk
            out["misses"][t, l] = mi
            out["proactive"][t, l] = pro
            out["margins"][t, l] = min(ref_margin, m_acc)
            out["certified"][t, l] = ref_margin >= tol and m_acc >= tol
            out["counters"][l] += np.array([K - mi, mi, pro], np.uint64)
            ref_margin = m_next if next_refines else np.inf
    bits = np.zeros((L, NW), np.uint32)
    for l in range(L):
        for e in np.flatnonzero(chains[l].in_cache):
            bits[l, e // 32] |= np.uint32(1 << (e % 32))
    out["cache_bits"] = bits
    out["aT"] = np.stack([c.aT for c in chains])
    return out


_W = None                   # the weights, set once per worker process


def _init_worker(W_bits):
    global _W
    _W = W_bits


def _stream_job(args):
    w, seed, b, tol, max_tries = args
    return _certify_stream(w, _W, seed, b, tol, max_tries)


def certified_streams(w, W_bits: np.ndarray, seed: int, streams, tol: float = 1e-3,
                      max_tries: int = 64, processes: int | None = None) -> dict:
    """Walk the given streams of workload w (weights W_bits [L][3N][d]) with
    redraws until every decision margin is >= tol; one worker process per
    stream (started with "spawn", so a caller that already holds a GPU
    context can use it), or in this process when processes == 1.

    Returns arrays stacked over the streams: attempts [S][T][L] (uint8, the
    generator's re-draw table), hidden [S][T][L][d] (bf16 bits), the fp64
    oracle's topk [S][T][L][K] (rank order), misses, proactive, margins,
    certified [S][T][L], cache_bits [S][L][NW], aT [S][L][N], counters
    [S][L][3], and the number of redraws per stream."""
    streams = list(streams)
    jobs = [(w, seed, b, tol, max_tries) for b in streams]
    n = min(len(streams), processes or default_threads())
    if n <= 1:
        _init_worker(W_bits)
        parts = [_stream_job(j) for j in jobs]
    else:
        ctx = multiprocessing.get_context("spawn")
        with ProcessPoolExecutor(max_workers=n, mp_context=ctx, initializer=_init_worker,
                                 initargs=(W_bits,)) as ex:
            parts = list(ex.map(_stream_job, jobs))
    res = {k: np.stack([q[k] for q in parts]) for k in parts[0] if k != "redraws"}
    res["redraws"] = np.array([q["redraws"] for q in parts])
    return res
