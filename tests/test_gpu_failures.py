"""Failure handling through the C ABI (needs a GB300): non-finite gradients
are reported by meq_sync and stay confined to their entry."""
import numpy as np
import pytest

from paper_2609_35701_gb300 import workloads as W

pytestmark = pytest.mark.gpu

LR, MU, WD, EPS = 0.02, 0.95, 0.1, 1e-7


@pytest.fixture(scope="module")
def meq():
    import __graft_entry__

    __graft_entry__.build()
    import torch

    assert torch.cuda.is_available()
    from paper_2609_35701_gb300 import meq as m

    return m


@pytest.mark.parametrize("bad,value", [(1, float("nan")), (2, float("inf")), (3, float("nan"))],
                         ids=["hidden_nan", "vector_inf", "remaining2d_nan"])
def test_nonfinite_gradient_reported_and_contained(meq, bad, value):
    """One element of entry `bad`'s step-0 gradient is non-finite. meq_sync
    reports MEQ_ERR_NONFINITE naming that entry, the report clears it, the
    next step reports it again (the momentum stays non-finite), and every
    other entry's parameters equal a clean run's bit for bit."""
    import torch

    shapes = [(256, 384), (384, 256), (1, 256), (300, 96)]
    kinds = [meq.HIDDEN, meq.HIDDEN, meq.VECTOR, meq.REMAINING_2D]
    wl = W.custom_workload(shapes, pattern="both", seed=19)
    outs = []
    for poison in (False, True):
        opt = meq.MeqMuon(shapes, kinds=kinds)
        params = [w.cuda() for w in W.initial_weights(wl)]
        for t in range(2):
            G = [g.cuda() for g in W.gradients(wl, t)]
            if poison and t == 0:
                G[bad].view(-1)[17] = value
            opt.step(params, G, LR, MU, WD, EPS)
            if poison:
                with pytest.raises(meq.MeqError) as e:
                    opt.sync()
                assert e.value.status == 4 and f"entry {bad}" in str(e.value), str(e.value)
                opt.sync()  # cleared by the report
            else:
                opt.sync()
        outs.append([p.cpu().numpy() for p in params])
        opt.close()
        torch.cuda.synchronize()
    clean, poisoned = outs
    for i in range(len(shapes)):
        if i == bad:
            assert not np.isfinite(poisoned[i]).all()
        else:
            assert np.array_equal(clean[i], poisoned[i]), i
