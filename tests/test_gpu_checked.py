"""The bounds-checked build (-DPCED_BOUNDS_CHECK): every guarded global index
(appended K/V row inside its layer region and below the capacity, partial
record slots, residual-stream rows, LM-head record tiles, selection rows) is
checked on the device; an index outside its buffer would set PCED_DEV_BOUNDS
and skip the access.  On valid inputs the checked library must report no
status bit and choose the same tokens with bit-identical hidden states as the
release library (the checks do not touch the arithmetic).  Slab and paged
caches, the max rule, MoE and a dynamic-beta first step are covered."""
import json
import os
import subprocess
import sys

import pytest

import checked_run

pytestmark = pytest.mark.gpu
HERE = os.path.dirname(os.path.abspath(__file__))


def test_checked_build_runs_clean_and_matches_release(cuda_ok):
    from paper_2601_08670_gb300 import build
    build.build(checked=True)
    env = dict(os.environ, PCED_LIB="checked")
    res = subprocess.run([sys.executable, os.path.join(HERE, "checked_run.py")], env=env, capture_output=True,
                         text=True, timeout=900)
    assert res.returncode == 0, res.stderr[-3000:]
    checked = json.loads(res.stdout.strip().splitlines()[-1])
    release = checked_run.run_cases()
    assert len(checked) == len(release) == len(checked_run.CASES)
    for c, r in zip(checked, release):
        assert c["case"] == r["case"]
        assert c["status"] == 0 and r["status"] == 0, (c, r)
        assert c["tokens"] == r["tokens"], c["case"]
        assert c["hidden"] == r["hidden"], c["case"]
