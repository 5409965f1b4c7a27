"""The MONE_DEBUG build: the same library with device-side index checks (tile rows and
columns against their buffers, the 16-byte alignment of TMA coordinates).  A failed check
skips the access, latches DEV_CHECK and is reported by mone_mem_sync as MONE_ERR_CHECK;
nothing faults.  Here the debug library, loaded in a child process through MONE_LIB, runs
small workloads of every kernel family and must report no failed check and match the oracle."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

SCRIPT = r'''
import sys
sys.path.insert(0, sys.argv[1])
sys.path.insert(0, sys.argv[1] + "/tests")
import torch
import paper_2608_17616_gb300 as mone
import workloads as wk
from harness import DeviceRun, oracle_chain, oracle_read, gpu_layout, rel_fro
assert mone.LIB_PATH.endswith("libmone_debug.so"), mone.LIB_PATH
cases = [
    (wk.Workload("dbg_pair", 70, 1, 2, 256, 256, 256, 2, 64, 256, 2 * 256 + 40, 40, "bf16", wk.PAPER, 0.3), 2e-2),
    (wk.Workload("dbg_b2", 71, 1, 3, 256, 256, 256, 2, 64, 1024, 1024 + 100, 16, "bf16", wk.PLAIN, 0.3), 2e-2),
    (wk.Workload("dbg_one", 72, 1, 2, 256, 256, 256, 2, 64, 128, 3 * 128 + 10, 16, "bf16", wk.PAPER, 0.3,
                 loss="mse"), 2e-2),
    (wk.WORKLOADS["tiny_f32"].replace(N=4 * 128), 1e-4),
]
for wl, tol in cases:
    run = DeviceRun(wl)
    run.ttl_context()                 # mone_mem_sync inside raises on MONE_ERR_CHECK
    Xq = wk.query_inputs(wl, "cuda")
    Kg, Vg = run.generate_kv(Xq)
    W1, W2, _, _ = run.state()
    mone.mone_mem_sync(run.h)
    for c in range(wl.chains):
        st, _ = oracle_chain(run, c)
        o1, o2 = gpu_layout(wl, st.W)
        assert rel_fro(W1[c], o1) <= tol and rel_fro(W2[c], o2) <= tol, (wl.name, c)
        Ko, Vo = oracle_read(run, st, c, Xq)
        ctx, layer = divmod(c, wl.n_layers)
        assert rel_fro(Kg[ctx, layer].float(), Ko) <= tol and rel_fro(Vg[ctx, layer].float(), Vo) <= tol, wl.name
    run.close()
print("debug ok")
'''


def test_debug_build_reports_no_failed_check_and_matches_the_oracle():
    from paper_2608_17616_gb300 import build
    path = build.build(debug=True)
    env = dict(os.environ, MONE_LIB=path)
    r = subprocess.run([sys.executable, "-c", SCRIPT, ROOT], env=env, capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, r.stdout[-4000:] + r.stderr[-4000:]
    assert "debug ok" in r.stdout
