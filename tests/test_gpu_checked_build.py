"""The checked build (-DEBD_CHECKS: every global access whose index comes
from device data checks it, records EBD_ERR_BOUNDS and skips the access) run
in a fresh process on the guarded steps of tests/test_gpu_guards.py: status
clean, guard words intact, outputs bit-identical to the normal build's; and
a window-attention call whose row offsets overrun the step's rows reports
EBD_ERR_BOUNDS with every guard intact."""
import os
import subprocess
import sys

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_checked_build_matches_and_catches(tmp_path):
    from paper_2609_16450_gb300 import build as b
    from tests import checked_run
    lib = b.build(checked=True)
    out = tmp_path / "checked.npz"
    env = dict(os.environ, EBD_LIBRARY=lib, PYTHONPATH=ROOT)
    r = subprocess.run([sys.executable, "-m", "tests.checked_run", str(out)], cwd=ROOT, env=env,
                       capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-4000:]
    chk = dict(np.load(out))
    from paper_2609_16450_gb300 import _ebd as E
    assert chk["bounds/status"] == E.EBD_ERR_BOUNDS and chk["bounds/guards"]
    ref = checked_run.run_cases()   # the normal build, in this process
    for k, v in ref.items():
        if k.endswith("/status"):
            assert chk[k] == 0 and v == 0, k
        elif k.endswith("/guards"):
            assert chk[k] and v, k
        else:
            np.testing.assert_array_equal(chk[k], v, err_msg=k)
