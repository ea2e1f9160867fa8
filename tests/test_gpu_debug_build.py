"""The checking flavour of the library (compiled with -DCRC_DEBUG).

In it every index a kernel derives -- stream, layer, chain, token, ring slot,
tile row, the experts a step makes resident -- is checked against the bound
of the array it addresses before use; a failed check latches CRC_EDEVICE and
skips the access instead of touching memory (the stand-in for a memory
checker, which this pool does not offer).  Tiny, a CTA-pair Qwen3 slice, an
N = 32 slice and an update-only slice run on it -- the fused kernel with and
without its trace, the chunked two-kernel path, the router heads -- in a
child process; every error word must stay zero and every result must equal,
bit for bit, the product library's on the same inputs.
"""
import os
import subprocess
import sys

import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))


@pytest.fixture(scope="module")
def C():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2609_04895_gb300 import build
    build.build()
    from paper_2609_04895_gb300 import crc
    crc.load()
    return crc


def test_checking_build_runs_clean_and_equals_the_product(C, tmp_path):
    from paper_2609_04895_gb300 import build
    build.build(debug=True)
    out = tmp_path / "debug.npz"
    r = subprocess.run([sys.executable, os.path.join(HERE, "debug_build_cases.py"), str(out)],
                       capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-4000:]
    dbg = dict(np.load(out))
    sys.path.insert(0, HERE)
    try:
        import debug_build_cases
    finally:
        sys.path.remove(HERE)
    rel = debug_build_cases.run_cases(C)
    assert set(dbg) == set(rel)
    for k in sorted(dbg):
        if k.endswith("error"):
            assert int(dbg[k]) == 0, k
            assert int(rel[k]) == 0, k
        else:
            assert np.array_equal(dbg[k], rel[k]), k
