"""Helpers that compare the CUDA path with the fp64 oracle (test code only).

Tolerances (relative, fp64 arithmetic on both sides' outputs):
  MOMENTUM_TOL  1e-5   B_t (fp32 on the GPU)
  STATS_TOL     1e-4   r, c, gamma_r, gamma_c computed from the GPU's own U
  PARAM_TOL     1e-5   W_{t+1} given the GPU's own normalised update
Momentum and params are compared per element relative to max(|ref|, RMS of
the matrix): an element that is the difference of two O(RMS) fp32 terms
carries an absolute rounding error of order 1e-7 * RMS, so a pure
elementwise relative bound is not meaningful where the terms cancel.
  UPDATE_TOL    1e-2   final normalised update vs the oracle's, Frobenius
  READBACK_TOL  1e-5   the update meq_read_update reports vs the one the
                       parameters received (Eq. (14) solved for U~), Frobenius
  NEAR_TIE      0.1    relative CV gap under which the two sides may pick
                       different directions; the oracle's update under the
                       GPU's direction must then meet UPDATE_TOL
"""
from __future__ import annotations

import numpy as np

from oracle import meqmuon as O

MOMENTUM_TOL = 1e-5
STATS_TOL = 1e-4
PARAM_TOL = 1e-5
UPDATE_TOL = 1e-2
NEAR_TIE = 0.1
READBACK_TOL = 1e-5


def rel_frob(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    nb = np.linalg.norm(b)
    return float(np.linalg.norm(a - b) / nb) if nb > 0 else float(np.linalg.norm(a - b))


def max_rel(a, b, floor_frac=1e-3):
    """max |a - b| / max(|b|, floor_frac * rms(b)) elementwise."""
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    rms = np.sqrt(np.mean(b * b)) if b.size else 0.0
    den = np.maximum(np.abs(b), floor_frac * rms)
    den = np.where(den > 0, den, 1.0)
    return float(np.max(np.abs(a - b) / den)) if b.size else 0.0


def gpu_update_from_params(W0, W1, lr, wd, rho=O.RHO):
    """The normalised update the GPU applied, recovered from Eq. (14)."""
    return ((1.0 - lr * wd) * np.asarray(W0, np.float64) - np.asarray(W1, np.float64)) / (rho * lr)


def staged_update(U_gpu, direction, eps=O.DELTA):
    U = np.asarray(U_gpu, np.float64)
    return O.row_normalize(U, eps) if direction == O.ROW else O.col_normalize(U, eps)


def check_staged_stats(Ug, st_gpu, eps, out):
    """Eqs. (7), (8) staged on the GPU's own U; returns the oracle's CVs."""
    r_o, c_o = O.row_col_rms(Ug)
    gr_o = O.coefficient_of_variation(r_o, eps)
    gc_o = O.coefficient_of_variation(c_o, eps)
    out["r"] = max_rel(st_gpu["r"], r_o, floor_frac=1e-6)
    out["c"] = max_rel(st_gpu["c"], c_o, floor_frac=1e-6)
    out["gamma_r"] = abs(st_gpu["gamma_r"] - gr_o) / max(gr_o, 1e-6)
    out["gamma_c"] = abs(st_gpu["gamma_c"] - gc_o) / max(gc_o, 1e-6)
    for k in ("r", "c", "gamma_r", "gamma_c"):
        assert out[k] <= STATS_TOL, (k, out)
    return gr_o, gc_o


def check_muon_step(W0, G, B_prev, W1_gpu, B_gpu, U_gpu, st_gpu, lr, mu, wd, eps=O.DELTA, nesterov=False,
                    update_tol=UPDATE_TOL, Ut_gpu=None):
    """All checks of one matrix after one GPU step under the Muon rule,
    Eq. (6): momentum end to end, statistics and params staged on the GPU's
    own U, and the applied update U against the oracle's."""
    W0 = np.asarray(W0, np.float64)
    m, n = W0.shape
    W1_ora, B_ora, U_ora = O.moonlight_step(W0, np.asarray(G, np.float64), np.asarray(B_prev, np.float64), lr, mu,
                                            wd, nesterov=nesterov)
    out = {"momentum": max_rel(B_gpu, B_ora, floor_frac=1.0)}
    assert out["momentum"] <= MOMENTUM_TOL, out
    Ug = np.asarray(U_gpu, np.float64)
    check_staged_stats(Ug, st_gpu, eps, out)
    assert st_gpu["direction"] == 4, st_gpu["direction"]
    out["params_staged"] = max_rel(W1_gpu, O.moonlight_update(W0, Ug, lr, wd), floor_frac=1.0)
    assert out["params_staged"] <= PARAM_TOL, out
    applied = ((1.0 - lr * wd) * W0 - np.asarray(W1_gpu, np.float64)) / (lr * O.RHO * np.sqrt(max(m, n)))
    if Ut_gpu is not None:
        # meq_read_update reports sqrt(max(m, n)) U, the matrix Eq. (14) applied
        out["readback"] = rel_frob(np.asarray(Ut_gpu, np.float64) / np.sqrt(max(m, n)), applied)
        assert out["readback"] <= READBACK_TOL, out
        applied = np.asarray(Ut_gpu, np.float64) / np.sqrt(max(m, n))
    out["update"] = rel_frob(applied, U_ora)
    assert out["update"] <= update_tol, out
    return out, W1_ora, B_ora


def check_step(W0, G, B_prev, W1_gpu, B_gpu, U_gpu, st_gpu, lr, mu, wd, eps=O.DELTA, nesterov=False,
               update_tol=UPDATE_TOL, report=None, Ut_gpu=None):
    """All checks of one matrix after one GPU step. Returns a dict of errors.
    Ut_gpu: the update meq_read_update reported; it must equal the one the
    parameters received and is then the one compared with the oracle."""
    W0 = np.asarray(W0, np.float64)
    W1_ora, B_ora, info = O.hidden_step(W0, np.asarray(G, np.float64), np.asarray(B_prev, np.float64), lr, mu, wd,
                                        eps=eps, nesterov=nesterov)
    out = {}
    # momentum, Eq. (10)
    out["momentum"] = max_rel(B_gpu, B_ora, floor_frac=1.0)
    assert out["momentum"] <= MOMENTUM_TOL, out
    Ug = np.asarray(U_gpu, np.float64)
    gr_o, gc_o = check_staged_stats(Ug, st_gpu, eps, out)
    d_staged = O.select_direction(gr_o, gc_o)
    if d_staged != st_gpu["direction"]:
        assert abs(gr_o - gc_o) <= 2 * STATS_TOL * max(gr_o, gc_o) + 1e-6, ("staged direction", out)
    # params staged on the GPU's own update, Eq. (14)
    Ut_staged = staged_update(Ug, st_gpu["direction"], eps)
    W1_staged = O.apply_update(W0, Ut_staged, lr, wd)
    out["params_staged"] = max_rel(W1_gpu, W1_staged, floor_frac=1.0)
    assert out["params_staged"] <= PARAM_TOL, out
    # final update vs the oracle (end to end), with the near-tie rule
    applied = gpu_update_from_params(W0, W1_gpu, lr, wd)
    if Ut_gpu is None:
        Ut_gpu = applied
    else:
        out["readback"] = rel_frob(Ut_gpu, applied)
        assert out["readback"] <= READBACK_TOL, out
    ref = info["U_tilde"]
    out["flip"] = 0
    if st_gpu["direction"] != info["direction"]:
        gap = abs(info["gamma_r"] - info["gamma_c"]) / max(info["gamma_r"], info["gamma_c"], 1e-12)
        assert gap < NEAR_TIE, ("direction differs outside the near-tie band", gap, out)
        ref, _ = O.equilibrate_hidden(info["U"], eps, force_direction=st_gpu["direction"])
        out["flip"] = 1
    out["update"] = rel_frob(Ut_gpu, ref)
    out["ns_output"] = rel_frob(Ug, info["U"])
    assert out["update"] <= update_tol, out
    if report is not None:
        report.append(out)
    return out, W1_ora, B_ora, info
