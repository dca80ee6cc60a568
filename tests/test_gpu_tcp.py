"""The persistent tensor-core kernel (tcp) on the tc kernel's task records:
one CTA per SM streams X and the block values through rings across units,
bf16 with A in shared memory, fp32 (3xTF32) with A copied into tensor memory,
MMAs from per-stage programs built at create time. It runs a call only when
BSR_TCP=1 (it measured slower than the tc kernel on most shapes), so a
subprocess started with that setting sweeps every tc block shape against the
oracle at the fp32 / bf16 tolerance."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.parametrize("env", [{}, {"BSR_TCP_G": "1"}, {"BSR_TCP_G": "2"}])
def test_tcp_forced_on_every_tc_shape(env):
    e = dict(os.environ, BSR_TCP="1", BSR_TC_F32_R16="1", **env)
    r = subprocess.run([sys.executable, "-m", "tests.tcp_forced_check"], cwd=ROOT, env=e, capture_output=True,
                       text=True, timeout=900)
    assert r.returncode == 0, r.stdout[-4000:] + r.stderr[-2000:]
    assert r.stdout.count(": ok") == r.stdout.count("\n")
