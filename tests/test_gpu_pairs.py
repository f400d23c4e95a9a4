"""The grouped GEMM on CTA pairs (tcgen05.mma.cta_group::2, 256-row tiles),
on two pairs per cluster sharing their A rows by multicast, and on single
CTAs compute the same layer.

By default the shape decides (tall groups take pairs); EC2MOE_GEMM_PAIR=1
forces pairs wherever the epilogue allows them (also on short, ragged and
empty groups) and EC2MOE_GEMM_PAIR=0 forbids them; EC2MOE_GEMM_QUAD=1 runs
every pair GEMM with 256-column tiles and an even N-tile count as two pairs
per cluster.  The variables are read once per process, so each setting runs
the layer parity tests in a child process.
"""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

SELECT = ("test_layer_forward or test_experts_and_combine_entry_points or test_zero_token_experts_and_tail_tiles "
          "or test_layer_is_deterministic")


MODES = {
    "pairs-forced": {"EC2MOE_GEMM_PAIR": "1"},
    "pairs-off": {"EC2MOE_GEMM_PAIR": "0"},
    "quad": {"EC2MOE_GEMM_QUAD": "1"},
    "quad-pairs-forced": {"EC2MOE_GEMM_PAIR": "1", "EC2MOE_GEMM_QUAD": "1"},
}


@pytest.mark.parametrize("mode", sorted(MODES))
def test_layer_parity_with_pair_gemm_setting(mode):
    env = dict(os.environ, **MODES[mode])
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-m", "gpu", "-p", "no:cacheprovider",
                        os.path.join(ROOT, "tests", "test_gpu_parity.py"), "-k", SELECT],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=1500)
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-2000:]


def test_zero_wait_budget_on_two_pair_clusters():
    """A timeout inside the two-pair cluster GEMM (every wait given a zero
    budget) ends with EC2MOE_ERR_TIMEOUT and a context that still runs the
    layer to the same output, as for the other kernel families."""
    env = dict(os.environ, EC2MOE_GEMM_QUAD="1")
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-m", "gpu", "-p", "no:cacheprovider",
                        os.path.join(ROOT, "tests", "test_gpu_failure.py"), "-k", "mixtral-pairs"],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-2000:]

