"""Cases run on both flavours of the library by test_gpu_debug_build.py.

Run as a script, it loads the checking flavour (_build/debug/libcrc.so,
compiled with -DCRC_DEBUG), runs every case and saves the results to the
.npz file named on the command line; imported, ``run_cases`` runs them on
whichever library the binding has loaded.
"""
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import crc_synth as S  # noqa: E402

CASES = {
    "tiny": S.TINY,
    "pairs-n128": S.QWEN3_30B.with_(B=4, T=300, L=3, d=256),
    "n32": S.GPT_OSS_20B.with_(B=8, T=150, L=3, d=576),
    "r0-one-cta": S.QWEN3_30B.with_(B=3, T=70, L=2, R=0, C=16, d=256),
}


def run_cases(C) -> dict:
    import torch
    out = {}
    for name, w in CASES.items():
        p = C.problem_of(w)
        W = C.synth_weights(w.L, w.N, w.d, seed=51)
        h, _ = C.synth_hidden(w.B, w.T, w.L, w.d, seed=52, rho_t=w.rho_t, rho_l=w.rho_l)
        heads = 3 if w.R > 0 else 2
        runs = {}
        # the fused kernel without and with its trace
        wsf = torch.empty(C.crc_fused_workspace_bytes(p), dtype=torch.uint8, device="cuda")
        st = C.State(p)
        C.route_and_cache(p, h, W, st, None, workspace=wsf)
        runs["fused"] = (st, None)
        st = C.State(p)
        tr = C.Trace.alloc(p, w.T, caches=True, rank_order=False, topk_set=True)
        C.route_and_cache(p, h, W, st, tr, workspace=wsf)
        runs["fused_traced"] = (st, tr)
        # the two-kernel path, traced in rank order, chunks of 7 tokens
        ws7 = torch.empty(C.crc_workspace_bytes(p, 7), dtype=torch.uint8, device="cuda")
        st = C.State(p)
        tr = C.Trace.alloc(p, w.T, caches=True, topk_set=True)
        C.route_and_cache(p, h, W, st, tr, workspace=ws7)
        runs["chunked"] = (st, tr)
        # router heads on their own
        sc = C.route_scores(p, h, W, heads=heads)
        out[f"{name}/scores"] = sc[:, :, :, :heads].cpu().numpy()   # the S slot is unset when R = 0
        out[f"{name}/device_error"] = np.array(C.crc_device_error())
        for rn, (st, tr) in runs.items():
            r = st.read(want_caches=True, want_retention=True, want_chain_counters=True)
            out[f"{name}/{rn}/error"] = np.array(r["error"])
            out[f"{name}/{rn}/cache_bits"] = r["cache_bits"]
            out[f"{name}/{rn}/counters"] = r["chain_counters"]
            out[f"{name}/{rn}/retention"] = r["retention"].view(np.uint32)
            if tr is not None:
                for k in ("topk", "topk_set", "misses", "proactive", "cache_mid", "cache_after"):
                    v = getattr(tr, k)
                    if v is not None:
                        out[f"{name}/{rn}/{k}"] = v.cpu().numpy()
    return out


if __name__ == "__main__":
    from paper_2609_04895_gb300 import build
    from paper_2609_04895_gb300 import crc as C
    C.load(build.build(debug=True))
    np.savez(sys.argv[1], **run_cases(C))
