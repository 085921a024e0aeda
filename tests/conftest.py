import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")
    config.addinivalue_line("markers", "slow: larger CPU case")


@pytest.fixture(scope="session")
def oracle():
    from oracle import oracle as o
    o.lib()
    return o


@pytest.fixture(scope="session")
def torch_philox(tmp_path_factory):
    """Philox4x32-10 blocks from PyTorch's header-only engine, run as a black
    box (an implementation independent of the oracle): f(seed, region_id,
    block_indices) -> (n, 4) uint32."""
    import subprocess
    import numpy as np
    pytest.importorskip("torch")
    from torch.utils.cpp_extension import include_paths
    exe = str(tmp_path_factory.mktemp("shim") / "torch_philox_shim")
    cmd = ["g++", "-std=c++17", "-O1", "-o", exe,
           os.path.join(ROOT, "tests", "helpers", "torch_philox_shim.cpp")]
    cmd += ["-I" + p for p in include_paths()]
    try:
        subprocess.check_call(cmd, stdout=subprocess.DEVNULL, stderr=subprocess.DEVNULL)
    except (subprocess.CalledProcessError, FileNotFoundError):
        pytest.skip("cannot compile against torch headers")

    def blocks(seed, region_id, idx):
        idx = np.asarray(idx, dtype=np.uint64).reshape(-1)
        lines = "\n".join("%d %d %d" % (seed, region_id, b) for b in idx)
        out = subprocess.run([exe], input=lines, capture_output=True, text=True,
                             check=True).stdout.split()
        return np.array(out, dtype=np.uint64).astype(np.uint32).reshape(-1, 4)
    blocks.exe = exe
    return blocks
