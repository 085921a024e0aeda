"""The debug-bounds build (libasmv_debug.so, ASMV_DEBUG_BOUNDS=1) on the GPU.

- On in-bounds tables it gives the bytes and statistics of the oracle (the
  checks change nothing): a mixed fill with ragged and unaligned payloads,
  a compare of a perturbed candidate and a restore.
- Its test hook makes the fill's payload loop run past the end of the
  payload while the allocation it checks against stays the table's: the
  call returns EBOUNDS and no byte past the allocation is written.  The
  region sits at the start of a device buffer much larger than the table
  says, so even a store the check failed to refuse would land inside memory
  this test owns.

Each case runs in a child process, which loads the debug build through the
ASMV_DEBUG_BOUNDS environment variable; this process checks the results
against the oracle."""
import json
import os
import subprocess
import sys

import numpy as np
import pytest

from paper_2608_20711_gb300 import workloads as W

from ._gpu import assert_stats_equal, oracle_fill_arena, oracle_region_stats, torch_cuda

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r'''
import json, sys
import numpy as np
sys.path.insert(0, sys.argv[1])
import torch
from paper_2608_20711_gb300 import asmv
from paper_2608_20711_gb300 import workloads as W
from tests.test_gpu_debug_bounds import table, BUF, PAYLOAD_ELEMS, GUARD, WIDEN
assert asmv.lib().asmv_debug_bounds() == 1
out = {}
ctx = asmv.Context(0)
# 1. fill, compare and restore of an in-bounds table
regs, size = table()
ref = torch.zeros(size, dtype=torch.uint8, device="cuda")
ctx.fill(asmv.regions_in_arena(regs, ref.data_ptr()), seed=11)
torch.cuda.synchronize()
cand = ref.clone()
rng = np.random.default_rng(5)
for r in regs:
    if r.dtype in W.FLOAT_DTYPES and r.n_elems > 1 and r.payload_offset % W.DTYPE_SIZE[r.dtype] == 0:
        W.perturb_sparse(cand, r, rng, rate=0.01)
host = cand.cpu().numpy()
for r in regs:                  # the unaligned payload: flip the low bit of a few bytes on the host
    if r.payload_offset % W.DTYPE_SIZE[r.dtype] != 0:
        idx = r.payload_offset + rng.choice(r.payload_bytes, 5, replace=False)
        host[idx] ^= 1
cand.copy_(torch.from_numpy(host))
st = ctx.compare(asmv.regions_in_arena(regs, ref.data_ptr()), asmv.regions_in_arena(regs, cand.data_ptr()),
                 W.DEFAULT_TOL)
snap = [torch.empty(max(1, r.payload_bytes), dtype=torch.uint8, device="cuda") for r in regs]
ctx.capture(asmv.regions_in_arena(regs, ref.data_ptr()), [s.data_ptr() for s in snap])
back = torch.full((size,), 0x33, dtype=torch.uint8, device="cuda")
ctx.restore(asmv.regions_in_arena(regs, back.data_ptr()), [s.data_ptr() for s in snap])
torch.cuda.synchronize()
np.save(sys.argv[2] + "/ref.npy", ref.cpu().numpy())
np.save(sys.argv[2] + "/cand.npy", cand.cpu().numpy())
np.save(sys.argv[2] + "/back.npy", back.cpu().numpy())
out["stats"] = st
# 2. the widened fill
buf = torch.full((BUF,), 0x5A, dtype=torch.uint8, device="cuda")
r = W.Region("w", "f32", PAYLOAD_ELEMS, "uniform", -1.0, 1.0, GUARD, GUARD, 0xA5, 7)
r.offset = 0
ctx.debug_widen(WIDEN)
try:
    ctx.fill(asmv.regions_in_arena([r], buf.data_ptr()), seed=3)
    out["widened_status"] = 0
except asmv.AsmvError as e:
    out["widened_status"] = e.status
ctx.debug_widen(0)
torch.cuda.synchronize()
np.save(sys.argv[2] + "/buf.npy", buf.cpu().numpy())
ctx.close()
print(json.dumps(out, default=float))
'''

BUF = 1 << 20
PAYLOAD_ELEMS = 16384            # 64 KiB of fp32
GUARD = 256
WIDEN = 16 << 10                 # the loop runs 16 KiB past the payload: still inside BUF


def table():
    """A small table over one arena: every fill distribution of the float
    formats and raw integers, ragged sizes, one unaligned payload."""
    specs = [("f32", "uniform", 1000), ("bf16", "normal", 7777), ("f16", "normal", 40001),
             ("f8e4m3", "normal", 12345), ("i32", "int_range", 3000), ("i8", "raw", 70001),
             ("f16", "uniform", 5)]
    regs = []
    for i, (dt, dist, n) in enumerate(specs):
        p0, p1 = {"uniform": (-2.0, 3.0), "normal": (0.0, 1.0), "int_range": (0, 1000),
                  "raw": (0, 0)}[dist]
        regs.append(W.Region("d%d" % i, dt, n, dist, p0, p1, 256 + 3 * (i == 2), 256, 0xA5, i))
    return regs, W.layout(regs) + 64


@pytest.fixture(scope="module")
def run(tmp_path_factory):
    torch_cuda()
    from paper_2608_20711_gb300 import build
    build.build(debug_bounds=True)
    d = str(tmp_path_factory.mktemp("dbg"))
    env = dict(os.environ, ASMV_DEBUG_BOUNDS="1")
    r = subprocess.run([sys.executable, "-c", CHILD, ROOT, d], env=env, capture_output=True, text=True,
                       timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-4000:]
    return json.loads(r.stdout.strip().splitlines()[-1]), d


def test_in_bounds_results_equal_the_oracle(run, oracle):
    out, d = run
    regs, size = table()
    ref = np.load(d + "/ref.npy")
    want = oracle_fill_arena(oracle, regs, size, 11)
    assert np.array_equal(ref, want)
    cand = np.load(d + "/cand.npy")
    for r, got in zip(regs, out["stats"]):
        assert_stats_equal(got, oracle_region_stats(oracle, ref, r, cand, r, W.DEFAULT_TOL), r.name)
    back = np.load(d + "/back.npy")
    for r in regs:                       # restore: payload back, guards rewritten with the canary
        a, b = r.offset, r.offset + r.alloc_bytes
        assert np.array_equal(back[a:b], want[a:b]), r.name


def test_widened_fill_is_refused_past_the_allocation(run, oracle):
    from paper_2608_20711_gb300 import asmv
    out, d = run
    assert out["widened_status"] == asmv.EBOUNDS
    buf = np.load(d + "/buf.npy")
    total = GUARD + 4 * PAYLOAD_ELEMS + GUARD
    assert np.all(buf[total:] == 0x5A)                # nothing written past the allocation
    r = W.Region("w", "f32", PAYLOAD_ELEMS, "uniform", -1.0, 1.0, GUARD, GUARD, 0xA5, 7)
    r.offset = 0
    want = oracle_fill_arena(oracle, [r], total, 3)
    assert np.array_equal(buf[:GUARD], want[:GUARD])
    assert np.array_equal(buf[GUARD:GUARD + 4 * PAYLOAD_ELEMS], want[GUARD:GUARD + 4 * PAYLOAD_ELEMS])
