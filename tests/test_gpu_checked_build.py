"""The checked build of the library (-DRPD_CHECKS): device-side bounds checks on the step's
indexed loads and stores (compact indices and canvas positions in the gather, split slots of
the head kernel's partials, rows and split counts in the merge) latch RPD_ERR_CHECK in the
step's status word and skip the access instead of trapping.  A set of parity tests runs
against librpd_checked.so in a child process: every output must still match the oracle and
no check may fire (the test helpers assert the status of every step)."""
import os
import subprocess
import sys

import pytest
import torch

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = os.path.join(ROOT, "paper_2609_36452_gb300")
CHECKED = os.path.join(PKG, "librpd_checked.so")
SUBSET = ("ragged or row_counts or tmem_ring or tilings_match or largest or empty or "
          "batched_matches or lazy_projection_small or layouts")


@pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")
def test_parity_subset_on_the_checked_build():
    subprocess.run([sys.executable, os.path.join(PKG, "_build.py"), "--checked"], check=True,
                   cwd=ROOT, timeout=900)
    env = dict(os.environ, RPD_LIBRARY=CHECKED)
    which = subprocess.run([sys.executable, "-c", "import paper_2609_36452_gb300 as r; print(r.lib_path)"],
                           cwd=ROOT, env=env, capture_output=True, text=True, check=True)
    assert which.stdout.strip() == CHECKED
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider",
                        "tests/test_gpu_parity.py", "-k", SUBSET],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=1500)
    assert r.returncode == 0, r.stdout[-4000:] + r.stderr[-2000:]
    summary = [line for line in r.stdout.splitlines() if " passed" in line][-1]
    print("checked build:", summary)
    assert int(summary.split(" passed")[0].split()[-1]) >= 40, summary
