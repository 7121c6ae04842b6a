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


@pytest.mark.parametrize("pair", [1, 0], ids=["cta_pair", "single_cta"])
def test_no_write_outside_buffers(meq, pair):
    """Ragged shapes of every parameter type, three steps: the guard bands
    around every workspace buffer keep their pattern, the caller's parameter
    buffers are not written outside their extent (guard bands of a sentinel
    value before and after each), and the gradients are not written at all."""
    import torch

    shapes = [(200, 333), (333, 200), (1, 7), (7, 1), (129, 385), (1, 300), (300, 90)]
    kinds = [meq.HIDDEN] * 5 + [meq.VECTOR, meq.REMAINING_2D]
    wl = W.custom_workload(shapes, pattern="both", seed=23)
    opt = meq.MeqMuon(shapes, kinds=kinds, debug_canaries=1, ns_cta_pair=pair)
    assert opt.canary_count > 2 * len(shapes)
    GB = 1024  # floats of guard on each side (keeps every view 16-byte aligned)
    sentinel = 12345.0

    def banded(ts):
        bufs, views = [], []
        for t in ts:
            b = torch.full((2 * GB + t.numel(),), sentinel, device="cuda")
            b[GB:GB + t.numel()] = t.reshape(-1).cuda()
            bufs.append(b)
            views.append(b[GB:GB + t.numel()].view(t.shape))
        return bufs, views

    pbufs, params = banded(W.initial_weights(wl))
    for t in range(3):
        gbufs, grads = banded(W.gradients(wl, t))
        before = [g.clone() for g in grads]
        opt.step(params, grads, LR, MU, WD, EPS)
        opt.sync()
        for b, g, g0, (r, c) in zip(gbufs, grads, before, shapes):
            assert torch.equal(g, g0)
            assert (b[:GB] == sentinel).all() and (b[GB + r * c:] == sentinel).all()
        for b, (r, c) in zip(pbufs, shapes):
            assert (b[:GB] == sentinel).all() and (b[GB + r * c:] == sentinel).all()
    opt.check_canaries()
    opt.close()


def test_canary_check_detects_a_change(meq):
    """The checker itself: a byte written into one guard band (from the host)
    is reported as MEQ_ERR_CORRUPTED."""
    shapes = [(128, 192), (192, 128)]
    wl = W.custom_workload(shapes, pattern="both", seed=3)
    opt = meq.MeqMuon(shapes, debug_canaries=1)
    params = [w.cuda() for w in W.initial_weights(wl)]
    opt.step(params, [g.cuda() for g in W.gradients(wl, 0)], LR, MU, WD, EPS)
    opt.sync()
    opt.check_canaries()
    meq.lib.meq_debug_corrupt_canary(opt._st, opt.canary_count // 2)
    with pytest.raises(meq.MeqError) as e:
        opt.check_canaries()
    assert e.value.status == 7
    opt.close()


def test_ns_gemm_stage_that_never_fills(meq):
    """debug_skip_load: in the first NS launch one operand stage is armed but
    half its bytes never come. The MMA issuer's bounded wait expires, every
    role of every CTA stops and drains (the MMA issuer waits for its issued
    MMAs before TMEM is freed), meq_sync reports MEQ_ERR_TIMEOUT and clears
    it, and the GPU context stays usable: a clean state then steps exactly as
    a clean state did before the fault."""
    import torch

    shapes = [(512, 768), (768, 512), (256, 256)]
    wl = W.custom_workload(shapes, pattern="both", seed=23)

    def clean_run():
        opt = meq.MeqMuon(shapes)
        params = [w.cuda() for w in W.initial_weights(wl)]
        for t in range(2):
            opt.step(params, [g.cuda() for g in W.gradients(wl, t)], LR, MU, WD, EPS)
        opt.sync()
        out = [p.cpu().numpy() for p in params]
        opt.close()
        return out

    before = clean_run()
    opt = meq.MeqMuon(shapes, debug_skip_load=1, wait_timeout_ms=200.0, use_graph=0)
    params = [w.cuda() for w in W.initial_weights(wl)]
    opt.step(params, [g.cuda() for g in W.gradients(wl, 0)], LR, MU, WD, EPS)
    with pytest.raises(meq.MeqError) as e:
        opt.sync()
    assert e.value.status == 5, str(e.value)  # MEQ_ERR_TIMEOUT
    opt.sync()  # cleared by the report
    opt.close()
    torch.cuda.synchronize()
    after = clean_run()
    for i in range(len(shapes)):
        assert np.array_equal(before[i], after[i]), f"matrix {i} differs after the timeout"


def test_debug_skip_load_validation(meq):
    with pytest.raises(meq.MeqError):
        meq.MeqMuon([(64, 64)], debug_skip_load=1, ns_cta_pair=0)
