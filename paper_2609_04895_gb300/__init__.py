"""GB300-native cache-aware MoE routing and expert residency.

The product is the CUDA library ``_build/libcrc.so`` (C ABI in
``include/crc.h``); :mod:`paper_2609_04895_gb300.crc` is its ctypes binding.
Build it with :func:`paper_2609_04895_gb300.build.build`.
"""
from . import crc  # noqa: F401
from .crc import (CrcError, State, Trace, cache_loss, cache_scan, load_time,  # noqa: F401
                  metrics, pinned_empty, problem, problem_of, route_and_cache,
                  route_and_cache_host, route_scores, synth_hidden, synth_weights,
                  transfer_plan, transfer_replay)

__all__ = ["crc", "CrcError", "State", "Trace", "cache_loss", "cache_scan", "load_time",
           "metrics", "pinned_empty", "problem", "problem_of", "route_and_cache",
           "route_and_cache_host",
           "route_scores", "synth_hidden", "synth_weights", "transfer_plan", "transfer_replay"]
