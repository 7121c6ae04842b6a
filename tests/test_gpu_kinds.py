"""Algorithm 1 over every parameter type on the GPU (hidden 2D weights, the
remaining 2D parameters via Eq. (12), 1D parameters via Eq. (13)) against
the fp64 oracle's param_step."""
import numpy as np
import pytest

import parity as PT
from oracle import meqmuon as O
from paper_2609_35701_gb300 import workloads as W

pytestmark = pytest.mark.gpu

LR, MU, WD, EPS = 0.02, 0.95, 0.1, 1e-7


@pytest.fixture(scope="module")
def meq():
    import __graft_entry__

    __graft_entry__.build()
    from paper_2609_35701_gb300 import meq as m

    return m


def run_kinds(meq, wl, steps, pick=None, **opts):
    import torch

    shapes = [(r, c) for _, r, c in wl.shapes]
    kinds = wl.kind_list()
    opt = meq.MeqMuon(shapes, kinds=kinds, **opts)
    params = [w.cuda() for w in W.initial_weights(wl)]
    idx = list(range(len(shapes))) if pick is None else pick
    Bp = {i: np.zeros(shapes[i]) for i in idx}
    cache = W.scale_table(wl)
    worst = {}
    for t in range(steps):
        G = W.gradients(wl, t, scale_cache=cache)
        W0 = {i: params[i].cpu().double().numpy() for i in idx}
        opt.step(params, [g.cuda() for g in G], LR, MU, WD, EPS)
        opt.sync()
        for i in idx:
            B = opt.read_momentum(i)
            W1 = params[i].cpu().numpy()
            st = opt.read_stats(i)
            if kinds[i] == O.HIDDEN:
                out, _, _, _ = PT.check_step(W0[i], G[i].double().numpy(), Bp[i], W1, B, opt.read_ns_output(i), st,
                                             LR, MU, WD, EPS, Ut_gpu=opt.read_update(i))
                err = out["update"]
            else:
                Wn, Bo, Ut = O.param_step(kinds[i], W0[i], G[i].double().numpy(), Bp[i], LR, MU, WD, eps=EPS)
                assert PT.max_rel(B, Bo, floor_frac=1.0) <= PT.MOMENTUM_TOL
                # the normalisation statistics (Eq. (7) of B and of N_r(B)) and
                # the parameters: fp32 arithmetic throughout, no NS
                Bd = B.astype(np.float64)
                r_o, _ = O.row_col_rms(Bd)
                assert PT.max_rel(st["r"][: r_o.size], r_o, 1e-6) <= PT.STATS_TOL
                if kinds[i] == O.REMAINING_2D:
                    _, c_o = O.row_col_rms(O.row_normalize(Bd, EPS))
                    assert PT.max_rel(st["c"], c_o, 1e-6) <= PT.STATS_TOL
                    assert st["direction"] == 2
                else:
                    assert st["direction"] == 3
                err = PT.max_rel(W1, Wn, floor_frac=1.0)
                assert err <= PT.PARAM_TOL, (i, kinds[i], err)
                assert PT.rel_frob(PT.gpu_update_from_params(W0[i], W1, LR, WD), Ut) <= 1e-5
                # Eq. (12) / (13) as meq_read_update reports it
                assert PT.rel_frob(opt.read_update(i), Ut) <= PT.READBACK_TOL
            worst[kinds[i]] = max(worst.get(kinds[i], 0.0), err)
            Bp[i] = B
    opt.close()
    return worst


def test_full_llama60m_every_parameter_type(meq):
    """All 58M parameters of Llama-60M in one state, 3 steps; embed / LM head,
    every RMSNorm weight and sampled hidden weights checked every step."""
    wl = W.get_workload("llama60m_full")
    names = [n for n, _, _ in wl.shapes]
    kinds = wl.kind_list()
    pick = [i for i, k in enumerate(kinds) if k != O.HIDDEN]
    pick += [names.index(f"layers.{l}.{m}") for l in (0, 7) for m in ("q_proj", "down_proj")]
    worst = run_kinds(meq, wl, 3, pick)
    assert set(worst) == {O.HIDDEN, O.REMAINING_2D, O.VECTOR}


def test_ragged_mixed_kinds(meq):
    """Odd sizes, tiny and zero-momentum entries of every type."""
    shapes = [(333, 77), (1, 5), (1, 1), (97, 130), (1000, 3), (200, 200), (1, 1027)]
    kinds = [O.REMAINING_2D, O.VECTOR, O.VECTOR, O.HIDDEN, O.REMAINING_2D, O.HIDDEN, O.VECTOR]
    wl = W.custom_workload(shapes, pattern="both", seed=31, kinds=kinds)
    run_kinds(meq, wl, 2)
