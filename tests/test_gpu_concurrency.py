"""Contexts from several host threads at once: each thread owns a context
and a stream (the library's model: a context per stream, not shared across
threads) and repeatedly fills and checks its own data while the others do
the same; the no-allocation compare runs from threads of its own.  Every
result must equal the oracle's, as it does when the calls run alone."""
import threading

import numpy as np
import pytest

from paper_2608_20711_gb300 import asmv

from ._gpu import assert_stats_equal, oracle_fill_arena, oracle_region_stats, torch_cuda
from .test_gpu_parity import TOL, _cmp_table, _perturb_host, _place

pytestmark = pytest.mark.gpu

THREADS = 4
ROUNDS = 5


def _case(oracle, seed):
    regs = _cmp_table(seed, n_regions=12)
    size = _place(regs)
    ref = oracle_fill_arena(oracle, regs, size, seed)
    cands = [_perturb_host(ref, regs, seed * 10 + j, dense=(j % 2 == 0)) for j in range(3)]
    want = [[oracle_region_stats(oracle, ref, r, c, r, TOL) for r in regs] for c in cands]
    return regs, size, ref, cands, want


def _worker(idx, case, errors, results):
    torch = torch_cuda()
    regs, size, ref, cands, want = case
    try:
        torch.cuda.set_device(0)
        stream = torch.cuda.Stream()
        ctx = asmv.Context(0)
        try:
            with torch.cuda.stream(stream):
                dref = torch.from_numpy(ref).to("cuda")
                dcs = [torch.from_numpy(c).to("cuda") for c in cands]
                scratch = torch.empty(size, dtype=torch.uint8, device="cuda")
            stream.synchronize()
            rr = asmv.regions_in_arena(regs, dref.data_ptr())
            cc = [asmv.regions_in_arena(regs, d.data_ptr()) for d in dcs]
            ss = asmv.regions_in_arena(regs, scratch.data_ptr())
            out = []
            for _ in range(ROUNDS):
                out.append(("batched", ctx.compare_batched(rr, cc, TOL, stream=stream)))
                out.append(("single", [ctx.compare(rr, cc[1], TOL, stream=stream)]))
                ctx.fill(ss, seed=1000 + idx, stream=stream)
                out.append(("self", ctx.compare(ss, ss, TOL, stream=stream)))
            stream.synchronize()
            results[idx] = (out, scratch.cpu().numpy())
        finally:
            ctx.close()
    except Exception as e:                      # reported by the main thread
        errors.append((idx, repr(e)))


def _noalloc_worker(idx, case, errors, results):
    torch = torch_cuda()
    regs, size, ref, cands, want = case
    try:
        torch.cuda.set_device(0)
        stream = torch.cuda.Stream()
        with torch.cuda.stream(stream):
            dref = torch.from_numpy(ref).to("cuda")
            dc = torch.from_numpy(cands[2]).to("cuda")
        stream.synchronize()
        rr = asmv.regions_in_arena(regs, dref.data_ptr())
        cc = asmv.regions_in_arena(regs, dc.data_ptr())
        results[idx] = [asmv.compare_noalloc(rr, cc, TOL, stream=stream) for _ in range(ROUNDS)]
    except Exception as e:
        errors.append((idx, repr(e)))


def test_contexts_on_threads_agree_with_the_oracle(oracle):
    torch_cuda()
    cases = [_case(oracle, 70 + i) for i in range(THREADS)]
    errors, results, nresults = [], [None] * THREADS, [None] * 2
    threads = [threading.Thread(target=_worker, args=(i, cases[i], errors, results))
               for i in range(THREADS)]
    threads += [threading.Thread(target=_noalloc_worker, args=(j, cases[j], errors, nresults))
                for j in range(2)]
    for t in threads:
        t.start()
    for t in threads:
        t.join(timeout=600)
    assert not errors, errors
    for i, (regs, size, ref, cands, want) in enumerate(cases):
        out, scratch = results[i]
        for kind, got in out:
            if kind == "batched":
                for j in range(3):
                    for r, g, w in zip(regs, got[j], want[j]):
                        assert_stats_equal(g, w, "thread %d cand %d %s" % (i, j, r.name))
            elif kind == "single":
                for r, g, w in zip(regs, got[0], want[1]):
                    assert_stats_equal(g, w, "thread %d single %s" % (i, r.name))
            else:
                for g in got:
                    assert g["mismatches"] == 0 and g["guard_bad_bytes"] == 0
        filled = oracle_fill_arena(oracle, regs, size, 1000 + i,
                                   base=np.zeros(size, np.uint8))
        for r in regs:
            a, b = r.offset, r.offset + r.alloc_bytes
            np.testing.assert_array_equal(scratch[a:b], filled[a:b], err_msg="thread %d %s" % (i, r.name))
    for j in range(2):
        regs, size, ref, cands, want = cases[j]
        for got in nresults[j]:
            for r, g, w in zip(regs, got, want[2]):
                assert_stats_equal(g, w, "noalloc %d %s" % (j, r.name))
