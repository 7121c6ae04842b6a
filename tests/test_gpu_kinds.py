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


def test_rows_columns_and_vectors_at_the_rms_threshold(meq):
    """The reading of Eq. (9) for rows / columns whose RMS does not exceed
    delta (scale 0, no update from them), on the branches without
    Newton-Schulz, where the momentum's rows are the gradient's: a remaining
    2D parameter with a row at RMS 5e-8 and one at 3e-7 (rescaled to unit
    RMS), a column that is tiny in every row (dropped by the second stage of
    Eq. (12)), and vectors at RMS 4e-8 and 2e-7 (Eq. (13)). One step from
    B = 0, parameters and statistics against the oracle."""
    import torch

    rng = np.random.default_rng(23)
    G = rng.standard_normal((96, 40)) * 0.01
    G[7] = 5e-8 * np.sign(rng.standard_normal(40))
    G[8] = 3e-7 * np.sign(rng.standard_normal(40))
    G[:, 11] = 1e-12
    G[8, 11] = 0.0   # else row 8's rescaling (about 3e6) would lift column 11 above delta
    gv1 = np.full((1, 64), 4e-8)
    gv2 = np.full((1, 64), -2e-7)
    Gs = [G.astype(np.float32), gv1.astype(np.float32), gv2.astype(np.float32)]
    kinds = [O.REMAINING_2D, O.VECTOR, O.VECTOR]
    shapes = [g.shape for g in Gs]
    W0 = [rng.standard_normal(s).astype(np.float32) * 0.02 for s in shapes]
    opt = meq.MeqMuon(shapes, kinds=kinds)
    params = [torch.from_numpy(w.copy()).cuda() for w in W0]
    opt.step(params, [torch.from_numpy(g).cuda() for g in Gs], LR, MU, WD, EPS)
    opt.sync()
    for i, k in enumerate(kinds):
        W1 = params[i].cpu().numpy()
        Wn, _, Ut = O.param_step(k, W0[i].astype(np.float64), Gs[i].astype(np.float64), np.zeros(shapes[i]), LR, MU,
                                 WD, eps=EPS)
        assert PT.max_rel(W1, Wn, floor_frac=1.0) <= PT.PARAM_TOL, i
        assert PT.rel_frob(opt.read_update(i), Ut) <= PT.READBACK_TOL, i
    Ut0 = opt.read_update(0)
    assert np.all(Ut0[7] == 0.0) and np.all(Ut0[:, 11] == 0.0)
    assert np.all(np.isfinite(Ut0[8])) and np.sqrt((Ut0[8] ** 2).mean()) > 0.1   # rescaled by about 1 / 3e-7
    assert np.all(opt.read_update(1) == 0.0)
    assert np.allclose(opt.read_update(2), -1.0, atol=1e-5)
    # decay only where nothing was rescaled
    d = (1 - LR * WD)
    assert np.array_equal(params[1].cpu().numpy(), (d * W0[1]).astype(np.float32)) or \
        PT.max_rel(params[1].cpu().numpy(), d * W0[1].astype(np.float64), floor_frac=1.0) <= PT.PARAM_TOL
    opt.close()
