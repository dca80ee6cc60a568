"""The SIMT kernel at every task size: the per-call chooser picks one task
size per product, so a subprocess started with BSR_XS_G forces each size in
turn (and with it the epilogue form: one, two or several warps per item, or
several items per warp for one-row blocks) and checks block shapes of both
dtypes against the oracle at the fp32 / bf16 tolerance."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.parametrize("G", ["1", "2", "3", "4", "6", "7", "12", "14", "24", "48", "96"])
def test_xs_forced_task_size(G):
    e = dict(os.environ, BSR_XS_G=G, BSR_FORCE_VARIANT="xstage")
    r = subprocess.run([sys.executable, "-m", "tests.xs_task_size_check"], cwd=ROOT, env=e, capture_output=True,
                       text=True, timeout=900)
    assert r.returncode == 0, r.stdout[-4000:] + r.stderr[-2000:]
    assert r.stdout.count(": ok") == r.stdout.count("\n")
