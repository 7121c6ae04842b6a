"""meq_step_prepare + meq_step_apply: the step split before the parameter
update (so a caller can overlap work on the previous parameters with the
next step's momentum, Newton-Schulz and statistics) equals meq_step."""
import numpy as np
import pytest
import torch

from paper_2609_35701_gb300 import workloads as W

pytestmark = pytest.mark.gpu

LR, MU, WD, EPS = 0.02, 0.95, 0.1, 1e-7


@pytest.fixture(scope="module")
def meq():
    import __graft_entry__

    __graft_entry__.build()
    assert torch.cuda.is_available()
    from paper_2609_35701_gb300 import meq as m

    return m


def _run(meq, wl, kinds, steps, split, **opts):
    shapes = [(r, c) for _, r, c in wl.shapes]
    opt = meq.MeqMuon(shapes, kinds=kinds, **opts)
    params = [w.contiguous().cuda() for w in W.initial_weights(wl)]
    cache = W.scale_table(wl)
    for t in range(steps):
        grads = [g.contiguous().cuda() for g in W.gradients(wl, t, scale_cache=cache)]
        if split:
            opt.step_prepare(grads, LR, MU, WD, EPS)
            opt.step_apply(params)
        else:
            opt.step(params, grads, LR, MU, WD, EPS)
    opt.sync()
    out = [p.cpu().numpy() for p in params]
    opt.close()
    return out


@pytest.mark.parametrize("use_graph", [1, 0])
def test_split_equals_step(meq, use_graph):
    shapes = [(200, 333), (333, 200), (768, 768), (1, 96), (64, 500)]
    kinds = [meq.HIDDEN, meq.HIDDEN, meq.HIDDEN, meq.VECTOR, meq.REMAINING_2D]
    wl = W.custom_workload(shapes, pattern="both", seed=21)
    a = _run(meq, wl, kinds, 3, False, use_graph=use_graph)
    b = _run(meq, wl, kinds, 3, True, use_graph=use_graph)
    for i, (x, y) in enumerate(zip(a, b)):
        assert np.array_equal(x, y), f"matrix {i}: split step differs from meq_step"


def test_split_protocol(meq):
    shapes = [(128, 256)]
    wl = W.custom_workload(shapes, seed=1)
    opt = meq.MeqMuon(shapes)
    p = [w.contiguous().cuda() for w in W.initial_weights(wl)]
    g = [x.contiguous().cuda() for x in W.gradients(wl, 0)]
    with pytest.raises(meq.MeqError):
        opt.step_apply(p)                      # no prepare pending
    opt.step_prepare(g, LR, MU, WD, EPS)
    with pytest.raises(meq.MeqError):
        opt.step_prepare(g, LR, MU, WD, EPS)   # second prepare before the apply
    with pytest.raises(meq.MeqError):
        opt.step(p, g, LR, MU, WD, EPS)        # meq_step while a prepare is pending
    opt.step_apply(p)
    opt.step(p, g, LR, MU, WD, EPS)            # back to whole steps
    opt.sync()
    opt.close()


def test_split_overlaps_a_copy_of_the_previous_params(meq):
    """The previous step's parameters, copied on another stream while the next
    prepare runs, are those of meq_step; the apply waits for the copy."""
    shapes = [(768, 2048), (2048, 768)]
    wl = W.custom_workload(shapes, pattern="row", seed=7)
    ref = []
    opt = meq.MeqMuon(shapes)
    params = [w.contiguous().cuda() for w in W.initial_weights(wl)]
    cache = W.scale_table(wl)
    for t in range(3):
        opt.step(params, [g.contiguous().cuda() for g in W.gradients(wl, t, scale_cache=cache)], LR, MU, WD, EPS)
        ref.append([p.cpu().numpy() for p in params])
    opt.close()

    opt = meq.MeqMuon(shapes)
    params = [w.contiguous().cuda() for w in W.initial_weights(wl)]
    host = [[torch.empty(p.shape, pin_memory=True) for p in params] for _ in range(3)]
    main, side = torch.cuda.current_stream(), torch.cuda.Stream()
    copied = torch.cuda.Event()
    for t in range(3):
        grads = [g.contiguous().cuda() for g in W.gradients(wl, t, scale_cache=cache)]
        opt.step_prepare(grads, LR, MU, WD, EPS)
        if t > 0:
            main.wait_event(copied)
        opt.step_apply(params)
        done = torch.cuda.Event()
        done.record(main)
        with torch.cuda.stream(side):
            side.wait_event(done)
            for h, p in zip(host[t], params):
                h.copy_(p, non_blocking=True)
            copied.record(side)
    torch.cuda.synchronize()
    opt.sync()
    opt.close()
    for t in range(3):
        for i in range(len(shapes)):
            assert np.array_equal(host[t][i].numpy(), ref[t][i]), f"step {t} matrix {i}"
