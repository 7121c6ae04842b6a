"""The allocation-free statistics entry point, meq_row_col_stats_noalloc.

It serves callers that cannot call cudaMalloc: code inside a framework that
owns all device memory through its own pool, and latency-critical paths that
must not allocate (cudaMalloc may synchronise the device). Its results are
compared with the fp64 oracle's statistics of the same matrix (Eqs. (7), (8),
(11)) and with the statistics the full optimizer step reports, on two calls
in a row that share the library's fixed scratch array.

Collected last on purpose: if it fails, a run that stops at the first failure
has already run every other test.
"""
import numpy as np
import pytest

import parity as PT
from oracle import meqmuon as O

pytestmark = pytest.mark.gpu

EPS, TIE = 1e-7, 1e-6


def _outputs(torch, m, n):
    r = torch.empty(m, dtype=torch.float32, device="cuda")
    c = torch.empty(n, dtype=torch.float32, device="cuda")
    g = torch.empty(2, dtype=torch.float64, device="cuda")
    d = torch.empty(1, dtype=torch.int32, device="cuda")
    return r, c, g, d


def _check_against_oracle(U64, r, c, g, d, what):
    r_o, c_o = O.row_col_rms(U64)
    gr_o = O.coefficient_of_variation(r_o, EPS)
    gc_o = O.coefficient_of_variation(c_o, EPS)
    assert PT.max_rel(r.cpu().numpy(), r_o, floor_frac=1e-6) <= PT.STATS_TOL, what
    assert PT.max_rel(c.cpu().numpy(), c_o, floor_frac=1e-6) <= PT.STATS_TOL, what
    gg = g.cpu().numpy()
    assert abs(gg[0] - gr_o) <= PT.STATS_TOL * max(gr_o, 1e-6), (what, gg[0], gr_o)
    assert abs(gg[1] - gc_o) <= PT.STATS_TOL * max(gc_o, 1e-6), (what, gg[1], gc_o)
    want = O.select_direction(gr_o, gc_o)
    if int(d.item()) != want:  # only a tie within the statistics tolerance may flip
        assert abs(gr_o - gc_o) <= 2 * PT.STATS_TOL * max(gr_o, gc_o) + TIE, what


def test_noalloc_stats_match_oracle_and_step_twice_in_a_row():
    import __graft_entry__

    __graft_entry__.build()
    import torch

    from paper_2609_35701_gb300 import meq
    from paper_2609_35701_gb300 import workloads as W

    wl = W.custom_workload([(300, 200), (256, 640), (777, 129), (5, 3)], pattern="both", seed=21)
    shapes = [(r, c) for _, r, c in wl.shapes]
    opt = meq.MeqMuon(shapes)
    params = [w.cuda() for w in W.initial_weights(wl)]
    opt.step(params, [g.cuda() for g in W.gradients(wl, 0)], 0.02, 0.95, 0.1, EPS)
    opt.sync()
    for i, (m, n) in enumerate(shapes):
        ref = opt.read_stats(i)
        Uh = opt.read_ns_output(i)
        U = torch.from_numpy(Uh).cuda()
        r, c, g, d = _outputs(torch, m, n)
        for call in range(2):
            for t in (r, c, g):
                t.fill_(float("nan"))
            d.fill_(-1)
            assert meq.row_col_stats_noalloc(U, r, c, g, d, eps=EPS, tie_atol=TIE) == 0
            torch.cuda.synchronize()
            _check_against_oracle(Uh.astype(np.float64), r, c, g, d, (i, call))
            assert PT.max_rel(r.cpu().numpy(), ref["r"], floor_frac=1e-6) <= PT.STATS_TOL, (i, call)
            assert PT.max_rel(c.cpu().numpy(), ref["c"], floor_frac=1e-6) <= PT.STATS_TOL, (i, call)
            gg = g.cpu().numpy()
            assert abs(gg[0] - ref["gamma_r"]) <= PT.STATS_TOL * max(ref["gamma_r"], 1e-6), (i, call)
            assert abs(gg[1] - ref["gamma_c"]) <= PT.STATS_TOL * max(ref["gamma_c"], 1e-6), (i, call)
            assert int(d.item()) == ref["direction"], (i, call)
    opt.close()


def test_noalloc_llama7b_shapes_and_size_limit():
    """The Llama-7B hidden shapes (the largest the fixed scratch takes for
    these widths), timed with CUDA events; a shape just past the limit is
    refused with its buffers sized to the shape, so nothing could run past
    them even if the size check were missing."""
    import __graft_entry__

    __graft_entry__.build()
    import torch

    from paper_2609_35701_gb300 import meq

    gen = torch.Generator().manual_seed(7)
    for m, n in ((4096, 11008), (11008, 4096), (4096, 4096)):
        rs = torch.exp(torch.empty(m, 1).uniform_(-2.0, 2.0, generator=gen))
        U_h = torch.randn(m, n, generator=gen) * rs
        U = U_h.cuda()
        r, c, g, d = _outputs(torch, m, n)
        for call in range(2):
            assert meq.row_col_stats_noalloc(U, r, c, g, d, eps=EPS, tie_atol=TIE) == 0
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        reps = 20
        for _ in range(reps):
            meq.row_col_stats_noalloc(U, r, c, g, d, eps=EPS, tie_atol=TIE)
        e1.record()
        torch.cuda.synchronize()
        print(f"noalloc stats {m}x{n}: {e0.elapsed_time(e1) / reps * 1e3:.1f} us per call")
        _check_against_oracle(U_h.double().numpy(), r, c, g, d, (m, n))
        del U
    # 8192 x 8192 needs 8192 * 8 + 256 * 8192 floats of scratch, above 2^21
    m = n = 8192
    U = torch.zeros(m, n, dtype=torch.float32, device="cuda")
    r, c, g, d = _outputs(torch, m, n)
    assert meq.row_col_stats_noalloc(U, r, c, g, d, eps=EPS, tie_atol=TIE) == 1  # MEQ_ERR_INVALID_ARG
    assert b"scratch" in meq.lib.meq_last_error(None)
    torch.cuda.synchronize()
