"""The allocation-free statistics entry point against the statistics the full
optimizer step reports. It serves callers that cannot call cudaMalloc: code
inside a framework that owns all device memory through its own pool, and
latency-critical paths that must not allocate (cudaMalloc may synchronise the
device). Two calls in a row share the library's fixed scratch array.

Collected last on purpose: if it fails, a run that stops at the first failure
has already run every other test.
"""
import numpy as np
import pytest

import parity as PT

pytestmark = pytest.mark.gpu


def test_noalloc_stats_match_the_step_twice_in_a_row():
    import __graft_entry__

    __graft_entry__.build()
    import torch

    from paper_2609_35701_gb300 import meq
    from paper_2609_35701_gb300 import workloads as W

    wl = W.custom_workload([(300, 200), (256, 640), (777, 129), (5, 3)], pattern="both", seed=21)
    shapes = [(r, c) for _, r, c in wl.shapes]
    opt = meq.MeqMuon(shapes)
    params = [w.cuda() for w in W.initial_weights(wl)]
    opt.step(params, [g.cuda() for g in W.gradients(wl, 0)], 0.02, 0.95, 0.1, 1e-7)
    opt.sync()
    for i, (m, n) in enumerate(shapes):
        ref = opt.read_stats(i)
        U = torch.from_numpy(opt.read_ns_output(i)).cuda()
        r = torch.empty(m, dtype=torch.float32, device="cuda")
        c = torch.empty(n, dtype=torch.float32, device="cuda")
        g = torch.empty(2, dtype=torch.float64, device="cuda")
        d = torch.empty(1, dtype=torch.int32, device="cuda")
        for call in range(2):
            for t in (r, c, g):
                t.fill_(float("nan"))
            d.fill_(-1)
            assert meq.row_col_stats_noalloc(U, r, c, g, d, eps=1e-7, tie_atol=1e-6) == 0
            torch.cuda.synchronize()
            assert PT.max_rel(r.cpu().numpy(), ref["r"], floor_frac=1e-6) <= PT.STATS_TOL, (i, call)
            assert PT.max_rel(c.cpu().numpy(), ref["c"], floor_frac=1e-6) <= PT.STATS_TOL, (i, call)
            gg = g.cpu().numpy()
            assert abs(gg[0] - ref["gamma_r"]) <= PT.STATS_TOL * max(ref["gamma_r"], 1e-6), (i, call)
            assert abs(gg[1] - ref["gamma_c"]) <= PT.STATS_TOL * max(ref["gamma_c"], 1e-6), (i, call)
            assert int(d.item()) == ref["direction"], (i, call)
    # sizes beyond the fixed scratch are rejected before any work is enqueued
    big = torch.empty(8, 1, dtype=torch.float32, device="cuda")
    assert meq.lib.meq_row_col_stats_noalloc(big.data_ptr(), 1 << 20, 1 << 12, 1e-7, 1e-6, big.data_ptr(),
                                             big.data_ptr(), big.data_ptr(), big.data_ptr(), None) == 1
    opt.close()
