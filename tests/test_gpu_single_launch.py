"""The one-launch NS (option ns_single_launch): every product of Eq. (5) in one
cooperative launch, tiles ordered by per-matrix completion counters.

Each output tile is computed by the same code from the same operands as in
the one-launch-per-product path, so the two paths must agree bit for bit;
the per-product path itself is checked against the oracle in
test_gpu_parity.py. A parity check against the oracle runs here too."""
import numpy as np
import pytest

import parity as PT
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


def _run(meq, wl, steps, **opts):
    shapes = [(r, c) for _, r, c in wl.shapes]
    opt = meq.MeqMuon(shapes, **opts)
    launches = opt.ns_gemm_launches_per_step
    params = [w.contiguous().cuda() for w in W.initial_weights(wl)]
    cache = W.scale_table(wl)
    for t in range(steps):
        grads = [g.contiguous().cuda() for g in W.gradients(wl, t, scale_cache=cache)]
        opt.step(params, grads, LR, MU, WD, EPS)
    opt.sync()
    out = [p.cpu().numpy() for p in params]
    mom = [opt.read_momentum(i) for i in range(len(shapes))]
    opt.close()
    return out, mom, launches


def _assert_same(a, b):
    for i, (x, y) in enumerate(zip(a, b)):
        assert np.array_equal(x, y), f"matrix {i} differs between the two NS launch schemes"


@pytest.mark.parametrize("shapes,ns_steps", [
    # two shape groups (transposed and not), ragged: 2 x 3 x 5 = 30 segments
    ([(200, 333), (333, 200), (200, 333)], 5),
    # Llama-130M's three groups (square, wide, tall), a few matrices each: 45 segments
    ([(768, 768)] * 6 + [(768, 2048)] * 3 + [(2048, 768)] * 3, 5),
    # five groups, three iterations: 5 x 3 x 3 = 45 segments
    ([(64, 64), (129, 385), (385, 129), (256, 1000), (1000, 64)], 3),
    # one matrix: every product waits on the previous one
    ([(256, 256)], 5),
    # several waves of tiles per product launch (Llama-130M-sized groups)
    ([(768, 768)] * 48 + [(768, 2048)] * 12, 5),
])
def test_single_launch_bitwise(meq, shapes, ns_steps):
    wl = W.custom_workload(shapes, pattern="both", seed=11)
    base, mom0, n0 = _run(meq, wl, 3, ns_steps=ns_steps)
    one, mom1, n1 = _run(meq, wl, 3, ns_steps=ns_steps, ns_single_launch=1)
    assert n0 == 3 * ns_steps and n1 == 1
    _assert_same(base, one)
    _assert_same(mom0, mom1)


def test_single_launch_graph_and_eager(meq):
    """Graph replay and eager enqueue of the one-launch NS agree."""
    wl = W.custom_workload([(512, 768), (768, 512)], pattern="row", seed=4)
    g, _, _ = _run(meq, wl, 2, ns_single_launch=1, use_graph=1)
    e, _, _ = _run(meq, wl, 2, ns_single_launch=1, use_graph=0)
    _assert_same(g, e)


def test_single_launch_falls_back(meq):
    """More segments than one launch holds: one launch per product again."""
    wl = W.custom_workload([(64 * (i + 1), 96 * (i + 1)) for i in range(4)], pattern="none", seed=2)
    _, _, n = _run(meq, wl, 1, ns_single_launch=1)   # 4 groups x 15 products > 48 segments
    assert n == 15
    _, _, n = _run(meq, wl, 1, ns_single_launch=1, ns_cta_pair=0)
    assert n == 15


def test_single_launch_parity(meq):
    """Staged parity against the fp64 oracle with the one-launch NS."""
    wl = W.custom_workload([(192, 320), (320, 192)], pattern="both", base_sigma=0.02, seed=3)
    shapes = [(r, c) for _, r, c in wl.shapes]
    opt = meq.MeqMuon(shapes, ns_single_launch=1)
    assert opt.ns_gemm_launches_per_step == 1
    params = [w.contiguous().cuda() for w in W.initial_weights(wl)]
    B_prev = [np.zeros(s) for s in shapes]
    cache = W.scale_table(wl)
    rep = []
    for t in range(2):
        Gs = W.gradients(wl, t, scale_cache=cache)
        W0 = [p.cpu().double().numpy() for p in params]
        opt.step(params, [g.contiguous().cuda() for g in Gs], LR, MU, WD, EPS)
        opt.sync()
        for i in range(len(shapes)):
            B = opt.read_momentum(i)
            PT.check_step(W0[i], Gs[i].double().numpy(), B_prev[i], params[i].cpu().numpy(), B,
                          opt.read_ns_output(i), opt.read_stats(i), LR, MU, WD, EPS, report=rep)
            B_prev[i] = B
    opt.close()
    assert len(rep) == 4
