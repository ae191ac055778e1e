"""Every attention kernel design (register gather, tcgen05 masked tiles, the
dense-suffix split where a case allows it) on the
same cases against the fp64 oracle, each forced in a fresh process (the design override is
read once per process)."""
import os
import subprocess
import sys

import pytest

from design_check import CASES

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))


@pytest.mark.parametrize("design", ["gather", "tile", "suffix"])
def test_design_matches_oracle(design):
    env = dict(os.environ, RIS_FORCE_DESIGN=design)
    r = subprocess.run([sys.executable, os.path.join(HERE, "design_check.py")], env=env, capture_output=True,
                       text=True, timeout=600)
    assert r.returncode == 0, r.stdout + r.stderr
    expected = sum(len(c[6]) if c[8] else 1 for c in CASES)
    assert r.stdout.count("max-abs") == expected, r.stdout
