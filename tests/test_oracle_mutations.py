"""Planted mistakes in a copy of the oracle must each fail at least one pin.

Every mutation is a plausible slip (a dropped term, a wrong sign, index or
normaliser, a transposed operand). The copy is a fresh module object; the
real oracle is not touched.
"""
import importlib.util
import os

import numpy as np
import pytest

import oracle_pins as P

ORACLE_PATH = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "oracle", "meqmuon.py")


def fresh_oracle():
    spec = importlib.util.spec_from_file_location("oracle_copy", ORACLE_PATH)
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def _ns_factory(variant):
    def ns(H, steps=5, coeffs=(3.4445, -4.7750, 2.0315)):
        a, b, c = coeffs
        H = np.asarray(H, np.float64)
        nrm = np.sqrt((H * H).sum()) if variant != "maxabs" else np.abs(H).max()
        if nrm == 0:
            return np.zeros_like(H)
        X = H / nrm
        for _ in range(steps if variant != "k4" else 4):
            if variant == "gram_transposed":
                A = X.T @ X
                X = a * X + X @ (b * A + c * A @ A) if X.shape[0] != X.shape[1] else a * X + (b * A + c * A @ A) @ X
                continue
            A = X @ X.T
            if variant == "swap_bc":
                X = a * X + (c * A + b * A @ A) @ X
            elif variant == "drop_a":
                X = (b * A + c * A @ A) @ X
            elif variant == "cubic":
                X = a * X + b * A @ X
            elif variant == "sign_b":
                X = a * X + (-b * A + c * A @ A) @ X
            else:
                X = a * X + (b * A + c * A @ A) @ X
        return X
    return ns


def _rms_swapped(X):
    X = np.asarray(X, np.float64)
    m, n = X.shape
    return np.sqrt((X * X).sum(1)) / np.sqrt(m), np.sqrt((X * X).sum(0)) / np.sqrt(n)


def _cv_sample(v, delta=1e-7):
    v = np.asarray(v, np.float64)
    k = v[v > delta]
    if k.size < 2:
        return 0.0
    return float(np.std(k, ddof=1) / k.mean())


def _cv_keep_zeros(v, delta=1e-7):
    v = np.asarray(v, np.float64)
    return float(np.std(v) / v.mean()) if v.mean() > 0 else 0.0


def _cv_mean_over_all(v, delta=1e-7):
    v = np.asarray(v, np.float64)
    k = v[v > delta]
    if k.size == 0:
        return 0.0
    mean = k.sum() / v.size
    return float(np.sqrt(((k - mean) ** 2).sum() / k.size) / mean)


MUTATIONS = {
    "ns_swap_bc": ("newton_schulz", _ns_factory("swap_bc")),
    "ns_drop_aX": ("newton_schulz", _ns_factory("drop_a")),
    "ns_cubic_only": ("newton_schulz", _ns_factory("cubic")),
    "ns_sign_b": ("newton_schulz", _ns_factory("sign_b")),
    "ns_four_steps": ("newton_schulz", _ns_factory("k4")),
    "ns_maxabs_normaliser": ("newton_schulz", _ns_factory("maxabs")),
    "ns_gram_transposed": ("newton_schulz", _ns_factory("gram_transposed")),
    "rms_sqrt_swapped": ("row_col_rms", _rms_swapped),
    "cv_sample_std": ("coefficient_of_variation", _cv_sample),
    "cv_keeps_zeros": ("coefficient_of_variation", _cv_keep_zeros),
    "cv_mean_over_all": ("coefficient_of_variation", _cv_mean_over_all),
    "select_flipped": ("select_direction", lambda gr, gc, tie_atol=1e-6: 0 if gr < gc else 1),
    "inverse_rms_no_threshold": ("_inverse_rms", lambda v, delta=1e-7: np.where(np.asarray(v, np.float64) > 0,
                                                                          1.0 / np.maximum(np.asarray(v, np.float64),
                                                                                           1e-300), 0.0)),
    "row_norm_multiplies": ("row_normalize", lambda X, delta=1e-7: np.asarray(X) * np.sqrt((np.asarray(X) ** 2).mean(1))[:, None]),
    "col_norm_uses_l2": ("col_normalize", lambda X, delta=1e-7: np.asarray(X) / np.maximum(np.linalg.norm(X, axis=0), 1e-300)[None, :]),
    "apply_no_decay": ("apply_update", lambda W, V, lr, wd, rho=0.2: np.asarray(W) - rho * lr * np.asarray(V)),
    "apply_sign": ("apply_update", lambda W, V, lr, wd, rho=0.2: (1 - lr * wd) * np.asarray(W) + rho * lr * np.asarray(V)),
    "apply_no_rho": ("apply_update", lambda W, V, lr, wd, rho=0.2: (1 - lr * wd) * np.asarray(W) - lr * np.asarray(V)),
    "apply_coupled_decay": ("apply_update", lambda W, V, lr, wd, rho=0.2: (1 - wd) * np.asarray(W) - rho * lr * np.asarray(V)),
    "momentum_damped": ("momentum_update", lambda Bp, G, mu: mu * np.asarray(Bp) + (1 - mu) * np.asarray(G)),
    "momentum_no_mu": ("momentum_update", lambda Bp, G, mu: np.asarray(Bp) + np.asarray(G)),
    "nesterov_wrong": ("ns_input", lambda B, G, mu, nesterov=False: np.asarray(B) + (mu * np.asarray(G) if nesterov else 0)),
    "two_sided_order_swapped": ("two_sided_normalize", lambda B, delta=1e-7: _col_then_row(B)),
    "vector_uses_l2": ("vector_normalize", lambda b, delta=1e-7: np.asarray(b) / np.linalg.norm(b)),
    "moonlight_sqrt_min": ("moonlight_update", lambda W, U, lr, wd, rho=0.2: (1 - lr * wd) * np.asarray(W)
                           - lr * rho * np.sqrt(min(np.shape(U))) * np.asarray(U)),
    "moonlight_no_shape_factor": ("moonlight_update", lambda W, U, lr, wd, rho=0.2: (1 - lr * wd) * np.asarray(W)
                                  - lr * rho * np.asarray(U)),
    "trajectory_skips_x0": ("ns_cv_trajectory", lambda H, steps=20, coeffs=None, delta=1e-7: _traj_shifted(H, steps)),
    "moonlight_coupled_decay": ("moonlight_update", lambda W, U, lr, wd, rho=0.2: (1 - wd) * np.asarray(W)
                                - lr * rho * np.sqrt(max(np.shape(U))) * np.asarray(U)),
}


def _traj_shifted(H, steps):
    """Trajectory that starts at X_1 instead of X_0 (an off-by-one)."""
    O = fresh_oracle()
    gr, gc = O.ns_cv_trajectory(H, steps + 1)
    return gr[1:], gc[1:]


def _col_then_row(B):
    B = np.asarray(B, np.float64)
    m, n = B.shape
    X = B / np.sqrt((B * B).sum(0, keepdims=True) / m)
    return X / np.sqrt((X * X).sum(1, keepdims=True) / n)


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_mutation_is_caught(name):
    pytest.importorskip("mpmath")
    attr, fn = MUTATIONS[name]
    O = fresh_oracle()
    setattr(O, attr, fn)
    failures = []
    for check in P.ALL_CHECKS:
        try:
            with np.errstate(all="ignore"):  # a planted mistake may overflow; the pins still judge it
                check(O)
        except Exception as e:  # AssertionError or a shape error from the mutation
            failures.append((check.__name__, type(e).__name__))
    assert failures, f"mutation {name} passed every pin"


def test_unmutated_copy_passes():
    pytest.importorskip("mpmath")
    O = fresh_oracle()
    for check in P.ALL_CHECKS:
        check(O)
