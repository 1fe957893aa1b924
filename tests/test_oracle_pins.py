"""The fp64 oracle against what the paper and the mathematics fix (no GPU)."""
import os
import subprocess
import sys

import numpy as np
import pytest

import oracle
from oracle_pins import PINS


@pytest.mark.parametrize("pin", PINS, ids=[p.__name__ for p in PINS])
def test_pin(pin):
    pin(oracle.default())


def test_thread_count_does_not_change_results():
    """OpenMP only splits independent output rows: 1 thread and many threads agree bitwise."""
    code = r"""
import sys, numpy as np
sys.path.insert(0, %r)
import oracle
rng = np.random.default_rng(5)
T, d, r, m = 64, 96, 8, 8
X, F, dY = rng.standard_normal((T, d)), rng.standard_normal((T, d)), rng.standard_normal((T, d))
W = [rng.standard_normal(s) * 0.2 for s in [(d, m), (m, r), (r, m), (m, d)]]
out = oracle.boundary_step(X, F, dY, *W)
np.savez(sys.argv[1], **out)
""" % os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    res = {}
    for n in ("1", "7"):
        path = "/tmp/oracle_threads_%s_%d.npz" % (n, os.getpid())
        env = dict(os.environ, OMP_NUM_THREADS=n)
        subprocess.run([sys.executable, "-c", code, path], check=True, env=env)
        res[n] = dict(np.load(path))
        os.remove(path)
    for k in res["1"]:
        np.testing.assert_array_equal(res["1"][k], res["7"][k], err_msg=k)
