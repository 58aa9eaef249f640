"""The traced build of the library (BANDLU_TRACE=1: the wide-band chain kernel records the
global timer at its panel boundaries and waits, include/bandlu_trace.h) factors exactly as
the production build does, and its timeline is consistent: every panel of the panel CTA is
stamped, in order, and each panel's events follow one another.  Runs in a child process,
which loads only the traced library; the production library reports no timeline."""
import json
import os
import subprocess
import sys

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = f"""
import os, sys, json
sys.path.insert(0, {ROOT!r})
sys.path.insert(0, os.path.join({ROOT!r}, "tests"))
import numpy as np, torch
from paper_2608_22099_gb300 import bandlu
import oracle
from gpu_helpers import DEV
lib = bandlu.load()
assert os.path.basename(lib._name) == "libbandlu_trace.so", lib._name
cap = bandlu.bandlu_trace_capacity()
n, kl, ku = 2048, 64, 64
ldab = 2 * kl + ku + 1
from paper_2608_22099_gb300.workloads import make_dense
A = make_dense(n, kl, ku, seed=41)
AB0 = oracle.dense_to_band(A.numpy(), kl, ku, ldab)
AB_ref, ipiv_ref, info_ref, _ = oracle.gbtrf(AB0, kl, ku)
AB = torch.from_numpy(np.ascontiguousarray(AB0)).to(DEV)
ipiv = torch.zeros(n, dtype=torch.int32, device=DEV)
info = torch.zeros(1, dtype=torch.int32, device=DEV)
assert bandlu.bandlu_trace_clear() == 0
assert bandlu.gbtrf(n, kl, ku, AB, ldab, ipiv, info) == 0
torch.cuda.synchronize()
same = bool(np.array_equal(AB.cpu().numpy().view(np.int64), AB_ref.view(np.int64))
            and np.array_equal(ipiv.cpu().numpy(), ipiv_ref) and int(info.item()) == info_ref)
T = np.zeros(4 * cap * 16, dtype=np.uint64)
assert bandlu.bandlu_trace_read(T, T.size) == 0
T = T.reshape(4, cap, 16).astype(np.int64)
print(json.dumps({{"cap": cap, "same": same, "a": T[0, :n // 4, :4].tolist(), "s1": T[1, :n // 4, :5].tolist()}}))
"""


def test_traced_build_factors_as_production_and_stamps_every_panel():
    env = dict(os.environ, BANDLU_TRACE="1")
    env.pop("BANDLU_CHECKED", None)
    r = subprocess.run([sys.executable, "-c", CHILD], cwd=os.path.join(ROOT, "tests"), env=env,
                       capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, (r.stdout[-3000:], r.stderr[-3000:])
    d = json.loads(r.stdout.strip().splitlines()[-1])
    assert d["cap"] == 8192
    assert d["same"], "traced build differs from the oracle"
    a = np.array(d["a"])   # panel CTA: start, step 2 sent, done, next block in
    npan = a.shape[0]
    assert (a[:, 0] > 0).all() and (np.diff(a[:, 0]) > 0).all()
    assert (a[:-1, 1] >= a[:-1, 0]).all() and (a[:-1, 2] >= a[:-1, 1]).all() and (a[:-1, 3] >= a[:-1, 2]).all()
    assert (a[:-1, 3] <= a[1:, 0]).all()
    s1 = np.array(d["s1"])  # streamer 1 (panel q on block q+1): in, first, wait, last, sent
    q = np.arange(npan - 1)
    assert (s1[q, 4] >= s1[q, 3]).all() and (s1[q, 3] >= s1[q, 1]).all()
    assert (a[q, 3] >= s1[q, 4]).all()  # A has block q+1 only after streamer 1 sent its band


def test_production_build_reports_no_timeline():
    from paper_2608_22099_gb300 import bandlu
    if os.environ.get("BANDLU_TRACE") == "1" or os.environ.get("BANDLU_CHECKED") == "1":
        pytest.skip("a development build is loaded in this process")
    assert bandlu.bandlu_trace_capacity() == 0
    buf = np.zeros(16, dtype=np.uint64)
    assert bandlu.bandlu_trace_read(buf, 16) != 0
