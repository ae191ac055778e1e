"""Every attention kernel design (register gather, TMA gather, tcgen05 masked tiles) on the
same cases against the fp64 oracle, each forced in a fresh process (the design override is
read once per process)."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))


@pytest.mark.parametrize("design", ["gather", "tma", "tile"])
def test_design_matches_oracle(design):
    env = dict(os.environ, RIS_FORCE_DESIGN=design)
    r = subprocess.run([sys.executable, os.path.join(HERE, "design_check.py")], env=env, capture_output=True,
                       text=True, timeout=600)
    assert r.returncode == 0, r.stdout + r.stderr
    assert r.stdout.count("max-abs") == 7
