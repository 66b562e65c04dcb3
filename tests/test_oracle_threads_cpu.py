"""The oracle's results do not depend on its OpenMP thread count: threads
only split independent vocabulary rows / output features, and every
reduction runs serially (CPU, subprocesses with 1 and 4 threads)."""
import os
import subprocess
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

SCRIPT = r"""
import sys, numpy as np
sys.path.insert(0, {root!r})
import oracle
from workloads import Config, make_inputs
cfg = Config("thr", 2, 3001, 192, 4, 6, 5, 14, "bf16", 0.7, 123)
x = make_inputs(cfg)
r = oracle.build_tree(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"], x["h0"])
np.savez({out!r}, threads=oracle.num_threads(), **{{k: v for k, v in r.items() if hasattr(v, "dtype")}})
"""


def run(threads, out):
    env = dict(os.environ, OMP_NUM_THREADS=str(threads))
    subprocess.run([sys.executable, "-c", SCRIPT.format(root=ROOT, out=str(out))], check=True, env=env,
                   capture_output=True, timeout=300)
    return np.load(out)


def test_oracle_is_bitwise_independent_of_thread_count(tmp_path):
    a = run(1, tmp_path / "t1.npz")
    b = run(4, tmp_path / "t4.npz")
    assert int(a["threads"]) == 1
    for k in a.files:
        if k == "threads":
            continue
        assert a[k].tobytes() == b[k].tobytes(), k
