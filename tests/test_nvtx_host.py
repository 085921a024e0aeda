"""Every C ABI call that launches work opens one NVTX range named after
itself, in the "asmv" domain, and closes it on every return path.  Checked
on the CPU: an NVTX injection library (tests/helpers/nvtx_probe.c) records
the ranges, and each call is made with arguments it rejects, so no GPU is
needed; the range must still open and close."""
import ctypes
import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HELPER = os.path.join(ROOT, "tests", "helpers", "nvtx_probe.c")

CALLS = ["asmv_fill", "asmv_guard_check", "asmv_compare", "asmv_compare_batched", "asmv_compare_eq",
         "asmv_compare_eq_digits", "asmv_restore", "asmv_capture", "asmv_compare_noalloc",
         "asmv_time_launches", "asmv_va_map", "asmv_va_unmap"]

CHILD = r'''
import ctypes, json, sys
sys.path.insert(0, sys.argv[1])
from paper_2608_20711_gb300 import asmv
L = asmv.lib()
P = ctypes.CDLL(sys.argv[2])
P.nvtx_probe_event.restype = ctypes.c_char_p
P.nvtx_probe_domain.restype = ctypes.c_char_p
n = ctypes.c_size_t(1)
null = None
rcs = {
    "asmv_fill": L.asmv_fill(null, null, n, ctypes.c_uint64(1), null),
    "asmv_guard_check": L.asmv_guard_check(null, null, n, null, null),
    "asmv_compare": L.asmv_compare(null, null, null, n, null, null, null),
    "asmv_compare_batched": L.asmv_compare_batched(null, null, null, ctypes.c_size_t(1), n, null, null, null),
    "asmv_compare_eq": L.asmv_compare_eq(null, null, null, ctypes.c_size_t(1), n, null, ctypes.c_double(0.9999),
                                         ctypes.c_double(1e-3), null, null, null),
    "asmv_compare_eq_digits": L.asmv_compare_eq_digits(null, null, null, ctypes.c_size_t(1), n, null, null, null,
                                                       null),
    "asmv_restore": L.asmv_restore(null, null, null, n, null),
    "asmv_capture": L.asmv_capture(null, null, null, n, null),
    "asmv_compare_noalloc": L.asmv_compare_noalloc(null, null, n, null, null, null),
    "asmv_time_launches": L.asmv_time_launches(L.asmv_time_launches.argtypes[0](), null, ctypes.c_int(0),
                                               ctypes.c_size_t(0), null, null, null),
    "asmv_va_map": L.asmv_va_map(ctypes.c_int(0), ctypes.c_uint64(0), ctypes.c_size_t(0), null),
    "asmv_va_unmap": L.asmv_va_unmap(null),
}
ev = [P.nvtx_probe_event(i).decode() for i in range(P.nvtx_probe_count())]
print(json.dumps({"rcs": rcs, "events": ev, "depth": P.nvtx_probe_depth(),
                  "max_depth": P.nvtx_probe_max_depth(), "domain": P.nvtx_probe_domain().decode()}))
'''


@pytest.fixture(scope="module")
def probe(tmp_path_factory):
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    inc = None
    for d in ("/usr/local/cuda/include", os.path.join(os.environ.get("CUDA_HOME", "/usr/local/cuda"), "include")):
        if os.path.exists(os.path.join(d, "nvtx3", "nvToolsExt.h")):
            inc = d
    if inc is None:
        pytest.skip("no NVTX3 headers")
    out = str(tmp_path_factory.mktemp("nvtx") / "libnvtx_probe.so")
    subprocess.run([cc, "-shared", "-fPIC", "-O1", "-I" + inc, HELPER, "-o", out], check=True)
    return out


def test_every_launching_call_opens_and_closes_one_range(probe):
    from paper_2608_20711_gb300 import build
    build.build()                      # rebuilds only when a source is newer than the library
    env = dict(os.environ, NVTX_INJECTION64_PATH=probe)
    r = subprocess.run([sys.executable, "-c", CHILD, ROOT, probe], env=env, capture_output=True, text=True,
                       timeout=120)
    assert r.returncode == 0, r.stderr
    import json
    out = json.loads(r.stdout.strip().splitlines()[-1])
    assert all(rc != 0 for rc in out["rcs"].values()), out["rcs"]      # every call rejected its arguments
    assert out["domain"] == "asmv"
    assert out["depth"] == 0 and out["max_depth"] == 1
    pushes = [e[1:] for e in out["events"] if e.startswith("+")]
    pops = [e for e in out["events"] if e.startswith("-")]
    assert pushes == CALLS, pushes
    assert len(pops) == len(pushes)
    # each push is closed before the next call's push
    seq = [e[0] for e in out["events"] if e[0] in "+-"]
    assert seq == ["+", "-"] * len(CALLS)
