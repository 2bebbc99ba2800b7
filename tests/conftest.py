import os
import subprocess
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA device (GB300, sm_103a)")
    config.addinivalue_line("markers", "slow: long-running test")


@pytest.fixture(scope="session")
def triton_philox(tmp_path_factory):
    """Returns f(seeds[S], ctr[S, N, 4]) -> outputs[S, N, 4] from Triton's own
    Philox under its CPU interpreter, run in a child process."""
    pytest.importorskip("triton")
    d = tmp_path_factory.mktemp("triton_philox")

    def run(seeds, ctr):
        src, dst = str(d / "in.npz"), str(d / "out.npy")
        np.savez(src, seeds=np.asarray(seeds, dtype=np.uint64), ctr=np.asarray(ctr, dtype=np.uint32))
        env = dict(os.environ, TRITON_INTERPRET="1", CUDA_VISIBLE_DEVICES="")
        script = os.path.join(ROOT, "tests", "triton_philox_ref.py")
        r = subprocess.run([sys.executable, script, src, dst], env=env, capture_output=True, text=True, timeout=600)
        if r.returncode != 0:
            pytest.skip(f"Triton interpreter unavailable: {r.stderr[-400:]}")
        return np.load(dst)

    return run


@pytest.fixture(params=[1, 8], ids=["pack1", "pack8"])
def packing_mode(request):
    """Runs a test under both probe packings, on the oracle and the library."""
    import oracle
    from paper_2609_38095_gb300 import build as zo_build
    from paper_2609_38095_gb300 import zo
    zo_build.build()
    with oracle.packing(request.param), zo.packing(request.param):
        yield request.param
